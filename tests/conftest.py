import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300) and the built extension")
    config.addinivalue_line("markers", "slow: longer CPU runs")


@pytest.fixture(autouse=True)
def guard_bands_intact(request):
    """After every GPU test: the guard bands around every live handle's
    activation buffers are intact, and no handle closed during the test found
    one overwritten (a kernel writing past a buffer fails the test that ran it)."""
    yield
    if request.node.get_closest_marker("gpu") is None:
        return
    binding = sys.modules.get("paper_2607_20293_gb300.binding")
    if binding is None or binding._lib is None:
        return
    import gc
    gc.collect()                                 # close handles the test dropped
    bad = [ev.cfg.get("n_emb") for ev in list(binding._live) if ev.check_guards() != binding.OK]
    failures, binding.guard_failures[:] = list(binding.guard_failures), []
    assert not bad and not failures, f"guard band overwritten: {bad} {failures}"
