"""The device-side failure path: every wait in the library's kernels is
bounded, and a wait that runs out records EVO_ERR_TIMEOUT in the handle's
status word instead of hanging the GPU.  The wait is made to run out in a
form that cannot fault: evo_test_wait_timeout runs the loop kernel's and the
tensor-core kernels' wait helpers in one thread of one block, on a barrier
that nothing arrives at, with a tiny limit (no cluster, no copy, no tensor
memory in flight).  The status must report the timeout once, and the next
ordinary call must succeed and match the oracle."""
import numpy as np
import pytest

from oracle import evo_oracle as O
from paper_2607_20293_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    import torch as _t
    if not _t.cuda.is_available():
        pytest.skip("no CUDA device")
    return _t


@pytest.fixture(scope="module")
def B(torch):
    from paper_2607_20293_gb300 import binding, build
    build.build()
    binding.load()
    return binding


@pytest.mark.parametrize("helper,limit", [(0, 10000), (1, 1000)])
def test_wait_runs_out_and_handle_recovers(torch, B, helper, limit):
    cfg = synth.config("tiny")
    W = synth.make_weights(cfg, 0)
    obs, noise = synth.make_obs(cfg, 1, 1), synth.make_noise(cfg, 1, 2)
    ev = B.Evo(cfg, W, 1)
    assert ev.status() == B.OK
    ev.test_wait_timeout(helper, limit)
    assert ev.status() == B.ERR_TIMEOUT
    assert ev.status() == B.OK                       # read and cleared
    S = synth.bernoulli_schedule(6, 10, 0.5, 3, force_t0=True)
    got = ev.denoise(torch.from_numpy(obs).cuda(), torch.from_numpy(noise).cuda(), S).cpu().numpy()
    assert ev.status() == B.OK
    assert float(np.max(np.abs(got - O.denoise(W, cfg, obs, noise, S)))) <= 1e-4


def test_wait_probe_rejects_unbounded_limits(torch, B):
    cfg = synth.config("tiny")
    ev = B.Evo(cfg, synth.make_weights(cfg, 0), 1)
    for helper, limit in [(0, 0), (0, 10**8), (1, 10**6), (2, 100)]:
        with pytest.raises(B.EvoError) as e:
            ev.test_wait_timeout(helper, limit)
        assert e.value.code == B.ERR_ARG
    assert ev.status() == B.OK
