"""evo_denoise_noalloc: the entry point for callers that cannot allocate device
memory when they run a query (code under CUDA stream capture, real-time
loops that forbid allocation after start-up, applications whose allocator owns
the device).  Its per-call scratch lives in the library's static device array,
so it must return what evo_denoise returns, call after call, and refuse sizes
that do not fit that array.

The file name makes pytest collect it last, after every other test."""

import numpy as np
import pytest

from paper_2607_20293_gb300 import synth

pytestmark = pytest.mark.gpu

TOL_BF16 = 3e-2


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


def test_noalloc_matches_denoise_on_consecutive_calls(torch, B):
    cfg = synth.config("pusht")
    n = 3
    W = synth.make_weights(cfg, 0)
    ev = B.Evo(cfg, W, n)
    S = synth.bernoulli_schedule(24, 100, 0.25, 11)
    for call in range(2):
        obs = torch.from_numpy(synth.make_obs(cfg, n, 40 + call)).cuda()
        noise = torch.from_numpy(synth.make_noise(cfg, n, 50 + call)).cuda()
        want = ev.denoise(obs, noise, S).cpu().numpy()
        out = torch.full((n, cfg["horizon"], cfg["action_dim"]), float("nan"), device="cuda")
        got = ev.denoise_noalloc(obs, noise, S, out).cpu().numpy()
        assert np.all(np.isfinite(got))
        assert float(np.max(np.abs(got - want))) <= TOL_BF16
    assert ev.status() == B.OK


def test_noalloc_rejects_sizes_beyond_the_static_array(torch, B):
    # one Push-T-shaped sample needs n_obs * (2L + 6) * E * 4 = 44 KiB of the 8 MiB array
    cfg = synth.config("pusht")
    n = 300
    ev = B.Evo(cfg, synth.make_weights(cfg, 0), n)
    obs = torch.zeros((n, cfg["n_obs"], cfg["obs_dim"]), device="cuda")
    noise = torch.zeros((cfg["n_steps"] + 1, n, cfg["horizon"], cfg["action_dim"]), device="cuda")
    out = torch.zeros((n, cfg["horizon"], cfg["action_dim"]), device="cuda")
    with pytest.raises(B.EvoError) as e:
        ev.denoise_noalloc(obs, noise, np.ones((24, 100), np.uint8), out)
    assert e.value.code == B.ERR_SHAPE
