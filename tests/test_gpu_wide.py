"""GPU parity of the batch-wide path (step-synchronous over all samples, the
projections and MLP on the tensor cores) against the float64 oracle.

The path is forced with a small `wide_rows` so that batches the oracle finishes
in seconds exercise it: several 128-row GEMM tiles, a ragged last tile, tiles
that mix lattices (population candidates with few samples each), both
empty-cache policies, coarse [L][T] lattices and device lattices.  Tolerance:
max-abs 3e-2 on final actions (bf16 mode)."""
import numpy as np
import pytest

from oracle import evo_oracle as O
from paper_2607_20293_gb300 import synth

from eq1_trace import check_reuse

pytestmark = pytest.mark.gpu

TOL = 3e-2


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


def check(got, want, what=""):
    got = np.asarray(got, np.float64)
    assert np.all(np.isfinite(got)), what
    err = float(np.max(np.abs(got - want)))
    assert err <= TOL, f"{what}: max-abs {err:.3e} > {TOL:g}"
    return err


def make(name, n, torch, B, seed=1, **kw):
    cfg = synth.config(name)
    W = synth.make_weights(cfg, 0)
    obs = synth.make_obs(cfg, n, seed)
    noise = synth.make_noise(cfg, n, seed + 1)
    ev = B.Evo(cfg, W, n, wide_rows=kw.pop("wide_rows", 1), **kw)
    return cfg, W, obs, noise, ev, torch.from_numpy(obs).cuda(), torch.from_numpy(noise).cuda()


@pytest.mark.parametrize("frac", [1.0, 0.125])
def test_wide_pusht_ragged_tiles(torch, B, frac):
    # 9 samples x 16 tokens = 144 rows: one full 128-row tile and a ragged one
    cfg, W, obs, noise, ev, d_obs, d_noise = make("pusht", 9, torch, B)
    S = synth.bernoulli_schedule(24, 100, frac, 21)
    got = ev.denoise(d_obs, d_noise, S).cpu().numpy()
    assert ev.last_call()["path"] == "wide"
    check(got, O.denoise(W, cfg, obs, noise, S), f"pusht f={frac}")


def test_wide_force_policy_and_zero_lattice(torch, B):
    cfg, W, obs, noise, ev, d_obs, d_noise = make("pusht", 3, torch, B, empty="force")
    S = synth.bernoulli_schedule(24, 100, 0.1, 22)
    S[:, 0] = 0                                   # t = 0 refreshes only through the policy
    check(ev.denoise(d_obs, d_noise, S).cpu().numpy(), O.denoise(W, cfg, obs, noise, S, "force"), "force")
    ev0 = B.Evo(cfg, W, 3, wide_rows=1)
    Z = np.zeros((24, 100), np.uint8)            # ZERO policy, nothing refreshed: the identity decoder
    check(ev0.denoise(d_obs, d_noise, Z).cpu().numpy(), O.denoise(W, cfg, obs, noise, Z), "zeros")
    assert ev0.last_call()["path"] == "wide"


def test_wide_layer_rows_and_device_lattice(torch, B):
    cfg, W, obs, noise, ev, d_obs, d_noise = make("pusht", 4, torch, B)
    S = synth.bernoulli_schedule(8, 100, 0.3, 23)           # coarse [L][T]
    got_h = ev.denoise(d_obs, d_noise, S).cpu().numpy()
    got_d = ev.denoise(d_obs, d_noise, torch.from_numpy(S).cuda()).cpu().numpy()
    check(got_h, O.denoise(W, cfg, obs, noise, S), "layer rows")
    assert np.array_equal(got_h, got_d)
    bad = S.copy()
    bad[2, 7] = 3
    out = torch.full((4, cfg["horizon"], cfg["action_dim"]), 5.0, device="cuda")
    with pytest.raises(B.EvoError) as e:                     # checked on the host before any launch
        ev.denoise(d_obs, d_noise, torch.from_numpy(bad).cuda(), out=out)
    assert e.value.code == B.ERR_SCHEDULE
    assert torch.all(out == 5.0)
    assert ev.status() == B.OK


def test_wide_matches_cluster_path(torch, B):
    # the same handle shape, both paths, one heterogeneous lattice: each within
    # tolerance of the oracle on a sample, and close to each other everywhere
    cfg, W, obs, noise, ev_w, d_obs, d_noise = make("manip", 16, torch, B)
    ev_c = B.Evo(cfg, W, 16, wide_rows=-1)
    S = synth.heterogeneous_schedule(24, 100, 24)
    gw = ev_w.denoise(d_obs, d_noise, S).cpu().numpy()
    gc = ev_c.denoise(d_obs, d_noise, S).cpu().numpy()
    assert ev_w.last_call()["path"] == "wide" and ev_c.last_call()["path"] == "cluster"
    idx = [0, 9, 15]
    want = O.denoise(W, cfg, obs[idx], noise[:, idx], S)
    check(gw[idx], want, "wide")
    check(gc[idx], want, "cluster")
    assert float(np.max(np.abs(gw - gc))) <= 2 * TOL


def test_wide_population_tiles_mix_lattices(torch, B):
    # 2 observations x 16 tokens = 32 rows per candidate: one 128-row tile holds
    # four lattices, so the GEMM's tile gate and the per-row refresh decide
    cfg = synth.config("pusht")
    W = synth.make_weights(cfg, 0)
    P, N = 6, 2
    obs, noise = synth.make_obs(cfg, N, 31), synth.make_noise(cfg, N, 32)
    pop = np.stack([synth.bernoulli_schedule(24, 100, f, 40 + i)
                    for i, f in enumerate([0.05, 0.6, 0.0, 0.3, 0.125, 1.0])])
    ev = B.Evo(cfg, W, (P + 1) * N, wide_rows=1)
    x, dev = ev.population(torch.from_numpy(obs).cuda(), torch.from_numpy(noise).cuda(), pop)
    assert ev.last_call()["path"] == "wide"
    x, dev = x.cpu().numpy(), dev.cpu().numpy()
    full = O.denoise(W, cfg, obs, noise, np.ones((24, 100), np.uint8))
    for p in range(P):
        want = O.denoise(W, cfg, obs, noise, pop[p])
        check(x[p], want, f"candidate {p}")
    ref_dev = np.linalg.norm((x - full[None]).reshape(P, N, -1), axis=2).mean(1)
    assert np.allclose(dev, ref_dev, atol=2 * TOL)
    assert dev[5] < 1e-6 * max(1.0, float(dev.max()))      # the all-ones candidate is the reference itself


@pytest.mark.parametrize("empty", ["zero", "force"])
def test_wide_population_edge_lattices(torch, B, empty):
    # lattices that differ by sample: each row is walked from its own lattice's
    # refreshed cells to its next one, so a lattice that refreshes only the very
    # first or the very last cell, only step 0, only the last step, or nothing
    # at all must still end at the oracle's actions
    cfg = synth.config("pusht")
    W = synth.make_weights(cfg, 0)
    U, T = 24, 100
    lat = np.zeros((6, U, T), np.uint8)
    lat[0, 0, 0] = 1                  # the first cell only
    lat[1, U - 1, T - 1] = 1          # the last cell only
    lat[2, :, 0] = 1                  # every unit at step 0, then skips to the end
    lat[3, :, T - 1] = 1              # every unit at the last step only
    lat[4, ::5, ::7] = 1              # a sparse grid
    P, N = lat.shape[0], 2            # lattice 5: nothing refreshed
    obs, noise = synth.make_obs(cfg, N, 51), synth.make_noise(cfg, N, 52)
    ev = B.Evo(cfg, W, (P + 1) * N, wide_rows=1, empty=empty)
    x, _ = ev.population(torch.from_numpy(obs).cuda(), torch.from_numpy(noise).cuda(), lat)
    assert ev.last_call()["path"] == "wide"
    x = x.cpu().numpy()
    for p in range(P):
        want = O.denoise(W, cfg, obs, noise, lat[p], policy=empty)
        check(x[p], want, f"lattice {p} ({empty})")


@pytest.mark.parametrize("force", [False, True])
def test_wide_trace_eq1_bitwise(torch, B, force):
    """bf16 caches on the batch-wide path: every skipped cell adds exactly the
    bf16 value stored at the unit's last refresh (Eq. 1), bit for bit, and a
    unit not refreshed yet adds zero (or, under FORCE, is computed at t = 0)."""
    kw = {"empty": "force"} if force else {}
    cfg, W, obs, noise, ev, d_obs, d_noise = make("pusht", 9, torch, B, **kw)
    S = synth.bernoulli_schedule(24, 100, 0.2, 23)
    if force:
        S[:, 0] = 0
    trace = torch.zeros((100, 24, 9, 16, 256), dtype=torch.float32, device="cuda")
    got = ev.denoise(d_obs, d_noise, S, trace=trace).cpu().numpy()
    assert ev.last_call()["path"] == "wide"
    assert check_reuse(trace.cpu().numpy(), S, bf16=True, force=force) > 100
    check(got, O.denoise(W, cfg, obs, noise, S, "force" if force else "zero"), "wide trace")


def test_repeated_calls_replay_the_captured_sequence(torch, B):
    """A call that repeats the previous one (same lattice, sizes and buffers) is
    captured into a CUDA graph and replayed: the first, second (captured) and
    third (replayed) calls give bit-identical actions; a new lattice, or new
    inputs in the same buffers, give that call's own result."""
    cfg, W, obs, noise, ev, d_obs, d_noise = make("pusht", 9, torch, B)
    out = torch.empty((9, 16, 2), device="cuda")
    S = synth.bernoulli_schedule(24, 100, 0.2, 31)
    runs = [ev.denoise(d_obs, d_noise, S, out=out).cpu().numpy() for _ in range(3)]
    assert ev.last_call()["path"] == "wide"
    assert np.array_equal(runs[0], runs[1]) and np.array_equal(runs[0], runs[2])
    check(runs[0], O.denoise(W, cfg, obs, noise, S), "replayed")
    S2 = synth.bernoulli_schedule(24, 100, 0.2, 32)
    got2 = ev.denoise(d_obs, d_noise, S2, out=out).cpu().numpy()
    check(got2, O.denoise(W, cfg, obs, noise, S2), "new lattice")
    assert not np.array_equal(got2, runs[0])
    obs3 = synth.make_obs(cfg, 9, 77)
    d_obs.copy_(torch.from_numpy(obs3))                 # same buffer, new contents
    for _ in range(3):
        got3 = ev.denoise(d_obs, d_noise, S2, out=out).cpu().numpy()
    check(got3, O.denoise(W, cfg, obs3, noise, S2), "new inputs in the same buffers")
    assert ev.status() == B.OK
