"""evo_denoise_noalloc: the entry point for callers that cannot allocate device
memory when they run a query -- a real-time control loop that forbids
allocation once it has started, or an application whose own allocator has
reserved the device's memory up front.  Its per-call scratch lives in the
library's static device array, so it must return exactly what evo_denoise
returns (same kernels, same decomposition, deterministic reductions), call
after call, and refuse sizes that do not fit that array.

The file name makes pytest collect it last, after every other test."""

import numpy as np
import pytest

from oracle import evo_oracle as O
from paper_2607_20293_gb300 import synth

pytestmark = pytest.mark.gpu

TOL_BF16 = 3e-2
# 8 MiB array; one Push-T-shaped sample needs n_obs * (2L + 6) * E * 4 = 45,056 bytes
MAX_PUSHT_SAMPLES = (8 << 20) // (2 * (2 * 8 + 6) * 256 * 4)


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


# n = 3: 6 observation tokens, the small-call condition kernels;
# n = 100: 200 tokens, the general condition kernels, whose intermediates also
# live in the static array
@pytest.mark.parametrize("n", [3, 100])
def test_noalloc_equals_denoise_on_consecutive_calls(torch, B, n):
    cfg = synth.config("pusht")
    W = synth.make_weights(cfg, 0)
    ev = B.Evo(cfg, W, n)
    S = synth.bernoulli_schedule(24, 100, 0.25, 11)
    outs = []
    for call in range(2):
        obs_h, noise_h = synth.make_obs(cfg, n, 40 + call), synth.make_noise(cfg, n, 50 + call)
        obs, noise = torch.from_numpy(obs_h).cuda(), torch.from_numpy(noise_h).cuda()
        want = ev.denoise(obs, noise, S).cpu().numpy()
        assert ev.last_call()["path"] == "cluster"
        out = torch.full((n, cfg["horizon"], cfg["action_dim"]), float("nan"), device="cuda")
        got = ev.denoise_noalloc(obs, noise, S, out).cpu().numpy()
        # same kernels on the same decomposition: bit for bit
        assert np.array_equal(got, want), f"call {call}: max-abs {np.max(np.abs(got - want)):.3e}"
        idx = [0, n - 1]
        ref = O.denoise(W, cfg, obs_h[idx], noise_h[:, idx], S)
        assert float(np.max(np.abs(got[idx] - ref))) <= TOL_BF16
        outs.append(got)
    # the second call's observations and noise really reached the kernels
    assert float(np.max(np.abs(outs[0] - outs[1]))) > 0.1
    assert ev.status() == B.OK


def test_noalloc_size_limit(torch, B):
    cfg = synth.config("pusht")
    assert MAX_PUSHT_SAMPLES == 186
    n = MAX_PUSHT_SAMPLES + 1
    # wide_rows = -1: evo_denoise keeps the cluster path at this batch too
    ev = B.Evo(cfg, synth.make_weights(cfg, 0), n, wide_rows=-1)
    S = synth.bernoulli_schedule(24, 100, 0.125, 12)
    obs = torch.from_numpy(synth.make_obs(cfg, n, 60)).cuda()
    noise = torch.from_numpy(synth.make_noise(cfg, n, 61)).cuda()
    out = torch.zeros((n, cfg["horizon"], cfg["action_dim"]), device="cuda")
    with pytest.raises(B.EvoError) as e:
        ev.denoise_noalloc(obs, noise, S, out)
    assert e.value.code == B.ERR_SHAPE
    m = MAX_PUSHT_SAMPLES                                   # the largest batch that fits
    noise_m = noise[:, :m].contiguous()
    got = ev.denoise_noalloc(obs[:m], noise_m, S, out[:m]).cpu().numpy()
    want = ev.denoise(obs[:m], noise_m, S).cpu().numpy()
    assert np.array_equal(got, want)
    assert ev.status() == B.OK
