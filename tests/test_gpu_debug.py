"""The debug build (EVO_DEBUG_CHECKS): device-side index checks at the main
global-memory accesses of the loop kernel and the batch-wide kernels record a
status bit and skip the access instead of trapping.  On valid inputs no check
fires -- the status stays OK -- and the checks change no arithmetic, so the
results equal the normal build's bit for bit, on both execution paths."""
import numpy as np
import pytest

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
    build.build(debug=True)
    binding.load()
    binding.load(debug=True)
    return binding


@pytest.mark.parametrize("name,n,kw", [("tiny", 1, {}), ("pusht", 2, {"wide_rows": -1}),
                                       ("pusht", 9, {"wide_rows": 1})])
def test_debug_build_checks_pass_and_results_match(torch, B, name, n, kw):
    cfg = synth.config(name)
    W = synth.make_weights(cfg, 0)
    obs = torch.from_numpy(synth.make_obs(cfg, n, 1)).cuda()
    noise = torch.from_numpy(synth.make_noise(cfg, n, 2)).cuda()
    S = synth.bernoulli_schedule(3 * cfg["n_layer"], cfg["n_steps"], 0.3, 5)
    outs = []
    for debug in (False, True):
        ev = B.Evo(cfg, W, n, debug_lib=debug, **kw)
        outs.append(ev.denoise(obs, noise, S).cpu().numpy())
        assert ev.last_call()["path"] == ("wide" if kw.get("wide_rows") == 1 else "cluster")
        assert ev.status() == B.OK
        assert ev.check_guards() == B.OK
        ev.close()
    assert np.array_equal(outs[0], outs[1])
