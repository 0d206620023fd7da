"""GPU parity of the redundancy-aware initialisation: the dissimilarity map of
Eq. 6 and its variants (evo_redundancy_map) and guided sampling (Eq. 7,
evo_guided_schedules) against the float64 oracle.

The map is compared on the same activations (the oracle's all-refresh trace,
and synthetic activations for the larger shapes) to 1e-5 absolute plus 1e-4
relative (fp32 sums of n products), and end to end from the GPU's own trace;
the schedules must be identical bit for bit (integer arithmetic)."""
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


@pytest.fixture(scope="module")
def tiny_trace():
    cfg = synth.config("tiny")
    W = synth.make_weights(cfg, 0)
    n = 3
    obs, noise = synth.make_obs(cfg, n, 11), synth.make_noise(cfg, n, 12)
    U, T = 3 * cfg["n_layer"], cfg["n_steps"]
    tr = {}
    O.denoise(W, cfg, obs, noise, np.ones((U, T), np.uint8), trace=tr)
    return cfg, W, obs, noise, O.trace_activations(tr, U, T)


def _close(got, want):
    got = np.asarray(got, np.float64)
    assert np.all(np.isfinite(got))
    assert np.allclose(got, want, atol=1e-5, rtol=1e-4), float(np.max(np.abs(got - want)))


@pytest.mark.parametrize("metric", ["cosine", "mse", "l1", "w1"])
def test_map_on_oracle_trace(torch, B, tiny_trace, metric):
    cfg, W, obs, noise, acts = tiny_trace
    trace = np.ascontiguousarray(acts.transpose(2, 1, 0, 3, 4), dtype=np.float32)   # [T][U][N][H][E]
    got = B.redundancy_map(torch.from_numpy(trace).cuda(), metric).cpu().numpy()
    _close(got, O.redundancy_map(trace.transpose(2, 1, 0, 3, 4).astype(np.float64), metric))


def test_map_end_to_end_from_gpu_trace(torch, B, tiny_trace):
    cfg, W, obs, noise, acts = tiny_trace
    U, T, H, E = 3 * cfg["n_layer"], cfg["n_steps"], cfg["horizon"], cfg["n_emb"]
    ev = B.Evo(cfg, W, 3)
    tr = torch.zeros((T, U, 3, H, E), device="cuda")
    ev.denoise(torch.from_numpy(obs).cuda(), torch.from_numpy(noise).cuda(), np.ones((U, T), np.uint8), trace=tr)
    got = B.redundancy_map(tr, "cosine").cpu().numpy()
    _close(got, O.redundancy_map(acts, "cosine"))


@pytest.mark.parametrize("metric", ["cosine", "w1"])
def test_map_push_t_sized_rows(torch, B, metric):
    # n = 16 x 256 entries per activation (Push-T-shaped), several chunks of the pair kernel
    rng = np.random.default_rng(21)
    T, U, N, n = 20, 4, 2, 4096
    base = rng.standard_normal((U, N, n))
    trace = (base[None] + 0.3 * rng.standard_normal((T, U, N, n))).astype(np.float32)
    got = B.redundancy_map(torch.from_numpy(trace).cuda(), metric).cpu().numpy()
    _close(got, O.redundancy_map(trace.transpose(2, 1, 0, 3).astype(np.float64), metric))


@pytest.mark.parametrize("metric", ["mse", "l1"])
def test_map_ragged_rows(torch, B, metric):
    # n = 77 entries: a partial chunk and rows that are not 16-byte multiples
    rng = np.random.default_rng(22)
    T, U, N, n = 7, 3, 2, 77
    trace = rng.standard_normal((T, U, N, n)).astype(np.float32)
    got = B.redundancy_map(torch.from_numpy(trace).cuda(), metric).cpu().numpy()
    _close(got, O.redundancy_map(trace.transpose(2, 1, 0, 3).astype(np.float64), metric))


def test_map_rejects_bad_shapes(torch, B):
    assert B.load().evo_redundancy_scratch_bytes(1, 4, 2, 64, 0) == 0          # T < 2
    assert B.load().evo_redundancy_scratch_bytes(10, 4, 2, 100, 3) == 0        # w1 needs a power of two
    assert B.load().evo_redundancy_scratch_bytes(10, 4, 2, 100, 0) > 0


@pytest.mark.parametrize("K,eps,gamma", [(120, 0.05, 2), (0, 0.05, 2), (800, 0.05, 2), (37, 0.0, 1), (300, 0.2, 3)])
def test_guided_schedules_bit_exact(torch, B, K, eps, gamma):
    d = synth.dissimilarity_map(8, 100, 5).astype(np.float32)
    P = 16
    rnd = synth.guided_randoms(P, max(K, 1), 7)
    got = B.guided_schedules(torch.from_numpy(d).cuda(), K, torch.from_numpy(rnd.view(np.int64)).cuda(),
                             eps, gamma).cpu().numpy()
    want = O.guided_schedules(d, K, eps, gamma, rnd)
    assert np.array_equal(got, want)
    assert np.all(got.reshape(P, -1).sum(1) == K)


def test_guided_schedules_zero_weights(torch, B):
    # eps = 0 with zero map entries: zero weights are drawn only when nothing else is left
    d = np.zeros((4, 10), np.float32)
    d[1, 3], d[2, 7] = 1.0, 0.5
    rnd = synth.guided_randoms(4, 5, 8)
    got = B.guided_schedules(torch.from_numpy(d).cuda(), 5, torch.from_numpy(rnd.view(np.int64)).cuda(), 0.0,
                             1).cpu().numpy()
    assert np.array_equal(got, O.guided_schedules(d, 5, 0.0, 1, rnd))
    assert np.all(got[:, 1, 3] == 1) and np.all(got[:, 2, 7] == 1)
