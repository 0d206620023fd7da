"""GPU parity: the CUDA path (through the C ABI) against the float64 oracle on
the same seeded inputs.

Tolerances (max-abs on final actions, normalised to [-1, 1]): 1e-4 in fp32
mode, 3e-2 in bf16 mode.  Small configs are compared element by element on
every sample; the large batched configs run at full size on the GPU, in the
launch configuration the benchmark uses, and are compared on a sample of
chunks that the oracle recomputes one by one (chunks are independent)."""
import numpy as np
import pytest

from oracle import evo_oracle as O
from paper_2607_20293_gb300 import synth

from eq1_trace import check_reuse

pytestmark = pytest.mark.gpu

TOL = {"fp32": 1e-4, "bf16": 3e-2}


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


def setup(name, n, torch, B, max_batch=None, **kw):
    cfg = synth.config(name)
    W = synth.make_weights(cfg, 0)
    obs = synth.make_obs(cfg, n, 1)
    noise = synth.make_noise(cfg, n, 2)
    ev = B.Evo(cfg, W, max_batch or n, **kw)
    return cfg, W, obs, noise, ev, torch.from_numpy(obs).cuda(), torch.from_numpy(noise).cuda()


def oracle_subset(W, cfg, obs, noise, S, idx, policy="zero"):
    return O.denoise(W, cfg, obs[idx], noise[:, idx], S, policy)


def check(got, want, tol, what=""):
    err = float(np.max(np.abs(np.asarray(got, np.float64) - want)))
    assert np.all(np.isfinite(got)), what
    assert err <= tol, f"{what}: max-abs {err:.3e} > {tol:g}"
    return err


# ------------------------------------------------------------------ tiny (fp32, DDIM)

@pytest.mark.parametrize("kind", ["bern_t0", "ones", "zeros", "bern", "layer_rows"])
@pytest.mark.parametrize("policy", ["zero", "force"])
def test_tiny_fp32(torch, B, kind, policy):
    cfg, W, obs, noise, ev, d_obs, d_noise = setup("tiny", 1, torch, B, empty=policy)
    U, T = 6, 10
    S = {"bern_t0": synth.bernoulli_schedule(U, T, 0.5, 3, force_t0=True),
         "ones": np.ones((U, T), np.uint8), "zeros": np.zeros((U, T), np.uint8),
         "bern": synth.bernoulli_schedule(U, T, 0.5, 8),
         "layer_rows": synth.bernoulli_schedule(2, T, 0.5, 9)}[kind]
    got = ev.denoise(d_obs, d_noise, S).cpu().numpy()
    want = O.denoise(W, cfg, obs, noise, S, policy)
    check(got, want, TOL["fp32"], f"tiny {kind} {policy}")


@pytest.mark.parametrize("cluster", [2, 4, 8])
def test_tiny_fp32_cluster_sizes(torch, B, cluster):
    cfg, W, obs, noise, ev, d_obs, d_noise = setup("tiny", 3, torch, B, cluster=cluster)
    S = synth.bernoulli_schedule(6, 10, 0.5, 3, force_t0=True)
    check(ev.denoise(d_obs, d_noise, S).cpu().numpy(), O.denoise(W, cfg, obs, noise, S), TOL["fp32"])


def test_tiny_bf16(torch, B):
    cfg = synth.config("tiny", dtype="bf16")
    W = synth.make_weights(cfg, 0)
    obs, noise = synth.make_obs(cfg, 2, 1), synth.make_noise(cfg, 2, 2)
    ev = B.Evo(cfg, W, 2)
    S = synth.bernoulli_schedule(6, 10, 0.5, 3, force_t0=True)
    got = ev.denoise(torch.from_numpy(obs).cuda(), torch.from_numpy(noise).cuda(), S).cpu().numpy()
    check(got, O.denoise(W, cfg, obs, noise, S), TOL["bf16"])


def test_tiny_trace_eq1(torch, B):
    """Skipped cells add exactly the stored cache; refreshed cells match the oracle's r."""
    cfg, W, obs, noise, ev, d_obs, d_noise = setup("tiny", 1, torch, B)
    U, T, H, E = 6, 10, cfg["horizon"], cfg["n_emb"]
    S = synth.bernoulli_schedule(U, T, 0.4, 21)
    trace = torch.zeros((T, U, 1, H, E), dtype=torch.float32, device="cuda")
    ev.denoise(d_obs, d_noise, S, trace=trace)
    tr = trace.cpu().numpy()
    otr = {}
    O.denoise(W, cfg, obs, noise, S, trace=otr)
    last = {}
    n_skip = 0
    for t in range(T):
        for b in range(U):
            refreshed, used = otr[(b, t)]
            want = np.zeros((1, H, E)) if used is None else used
            assert np.max(np.abs(tr[t, b] - want)) < 1e-4
            if S[b, t]:
                last[b] = tr[t, b].copy()
            elif b in last:
                assert np.array_equal(tr[t, b], last[b])      # bit-exact reuse of c_b
                n_skip += 1
            else:
                assert not tr[t, b].any()                     # reset cache contributes zero
    assert n_skip > 5


@pytest.mark.parametrize("name,n", [("tiny", 2), ("pusht", 1)])
def test_bf16_trace_eq1_bitwise(torch, B, name, n):
    """bf16 caches on the cluster path: every skipped cell adds exactly the bf16
    value stored at that unit's last refresh (Eq. 1), bit for bit."""
    cfg = synth.config(name, dtype="bf16")
    W = synth.make_weights(cfg, 0)
    obs, noise = synth.make_obs(cfg, n, 1), synth.make_noise(cfg, n, 2)
    ev = B.Evo(cfg, W, n, wide_rows=-1)
    U, T, H, E = 3 * cfg["n_layer"], cfg["n_steps"], cfg["horizon"], cfg["n_emb"]
    S = synth.bernoulli_schedule(U, T, 0.3, 22)
    trace = torch.zeros((T, U, n, H, E), dtype=torch.float32, device="cuda")
    got = ev.denoise(torch.from_numpy(obs).cuda(), torch.from_numpy(noise).cuda(), S, trace=trace).cpu().numpy()
    assert ev.last_call()["path"] == "cluster"
    assert check_reuse(trace.cpu().numpy(), S, bf16=True) > 20
    check(got, O.denoise(W, cfg, obs, noise, S), TOL["bf16"], name)


# ------------------------------------------------------------------ Push-T shaped (bf16, DDPM, batch 1)

@pytest.mark.parametrize("frac", [1.0, 0.5, 0.125])
def test_pusht_fractions(torch, B, frac):
    cfg, W, obs, noise, ev, d_obs, d_noise = setup("pusht", 1, torch, B)
    S = synth.bernoulli_schedule(24, 100, frac, 3)
    got = ev.denoise(d_obs, d_noise, S).cpu().numpy()
    check(got, O.denoise(W, cfg, obs, noise, S), TOL["bf16"], f"pusht f={frac}")


def _golden(task):
    import os
    path = os.path.join(os.path.dirname(__file__), "golden", f"schedules_{task}.txt")
    rows = [l for l in open(path) if l.strip() and not l.startswith("#")]
    return O.schedule_from_positions([(b, int(t)) for b, l in enumerate(rows) for t in l.split(";")[2].split()],
                                     24, 100)


@pytest.mark.parametrize("task", ["pusht", "kitchen"])
def test_pusht_published_schedule(torch, B, task):
    cfg, W, obs, noise, ev, d_obs, d_noise = setup("pusht", 1, torch, B)
    S = _golden(task)
    got = ev.denoise(d_obs, d_noise, S).cpu().numpy()
    check(got, O.denoise(W, cfg, obs, noise, S), TOL["bf16"], task)


@pytest.mark.parametrize("cluster", [4, 8, 16])
def test_pusht_cluster_sizes_and_device_lattice(torch, B, cluster):
    cfg, W, obs, noise, ev, d_obs, d_noise = setup("pusht", 2, torch, B, cluster=cluster)
    S = synth.bernoulli_schedule(8, 100, 0.3, 5)          # layer rows
    want = O.denoise(W, cfg, obs, noise, S)
    got_h = ev.denoise(d_obs, d_noise, S).cpu().numpy()
    got_d = ev.denoise(d_obs, d_noise, torch.from_numpy(S).cuda()).cpu().numpy()
    check(got_h, want, TOL["bf16"])
    assert np.array_equal(got_h, got_d)


def test_invalid_device_lattice_sets_status(torch, B):
    cfg, W, obs, noise, ev, d_obs, d_noise = setup("tiny", 1, torch, B)
    S = np.ones((6, 10), np.uint8)
    S[3, 4] = 7
    out = torch.full((1, cfg["horizon"], cfg["action_dim"]), 5.0, device="cuda")
    ev.denoise(d_obs, d_noise, torch.from_numpy(S).cuda(), out=out)
    assert ev.status() == B.ERR_SCHEDULE
    assert torch.all(out == 5.0)
    with pytest.raises(B.EvoError):
        ev.denoise(d_obs, d_noise, S, out=out)             # host lattice: rejected before launch
    assert ev.status() == B.OK


def test_odd_batch_with_two_samples_per_job(torch, B):
    cfg, W, obs, noise, ev, d_obs, d_noise = setup("pusht", 3, torch, B, job_samples=2)
    assert ev.launch_info()["job_samples"] == 2
    S = synth.bernoulli_schedule(24, 100, 0.25, 6)
    check(ev.denoise(d_obs, d_noise, S).cpu().numpy(), O.denoise(W, cfg, obs, noise, S), TOL["bf16"])


def test_handles_with_different_plans_coexist(torch, B):
    # one compiled shape, two shared-memory plans (100 and 10 loop steps): the
    # smaller handle, created second, must not shrink the larger one's launch limit
    big = setup("pusht", 1, torch, B)
    cfg_s = synth.config("pusht", n_steps=10)
    W_s = synth.make_weights(cfg_s, 0)
    obs_s, noise_s = synth.make_obs(cfg_s, 1, 1), synth.make_noise(cfg_s, 1, 2)
    ev_s = B.Evo(cfg_s, W_s, 1)
    cfg, W, obs, noise, ev, d_obs, d_noise = big
    S = synth.bernoulli_schedule(24, 100, 0.2, 8)
    S_s = synth.bernoulli_schedule(24, 10, 0.5, 9)
    for _ in range(2):
        got_s = ev_s.denoise(torch.from_numpy(obs_s).cuda(), torch.from_numpy(noise_s).cuda(), S_s).cpu().numpy()
        got = ev.denoise(d_obs, d_noise, S).cpu().numpy()
        check(got_s, O.denoise(W_s, cfg_s, obs_s, noise_s, S_s), TOL["bf16"], "10 steps")
        check(got, O.denoise(W, cfg, obs, noise, S), TOL["bf16"], "100 steps")


# ------------------------------------------------------------------ batched configs at full size

@pytest.mark.parametrize("path", ["wide", "cluster"])
def test_manip_batch64_heterogeneous(torch, B, path):
    cfg, W, obs, noise, ev, d_obs, d_noise = setup("manip", 64, torch, B, wide_rows=1024 if path == "wide" else -1)
    S = synth.heterogeneous_schedule(24, 100, 4)
    got = ev.denoise(d_obs, d_noise, S).cpu().numpy()
    assert ev.last_call()["path"] == path
    idx = [0, 17, 63]
    check(got[idx], oracle_subset(W, cfg, obs, noise, S, idx), TOL["bf16"], "manip")
    assert np.all(np.isfinite(got)) and np.all(np.abs(got) <= 1.5)


def test_automatic_decomposition_by_batch(torch, B):
    # with the cluster size left to the library, one handle holds the 16-, 8- and
    # 4-CTA decompositions and a call takes the one with the fewest job rounds
    cfg = synth.config("manip")
    W = synth.make_weights(cfg, 0)
    ev = B.Evo(cfg, W, 64)
    S = synth.heterogeneous_schedule(24, 100, 4)
    for n, C, idx in [(1, 16, [0]), (8, 8, [0, 7]), (64, 4, [0, 33, 63])]:
        obs, noise = synth.make_obs(cfg, n, 1), synth.make_noise(cfg, n, 2)
        got = ev.denoise(torch.from_numpy(obs).cuda(), torch.from_numpy(noise).cuda(), S).cpu().numpy()
        assert ev.last_call()["path"] == "cluster"
        assert ev.launch_info()["cluster"] == C, (n, ev.launch_info())
        check(got[idx], oracle_subset(W, cfg, obs, noise, S, idx), TOL["bf16"], f"batch {n}")
    assert ev.status() == B.OK


def test_scaleup_cluster_path_global_caches(torch, B):
    # n_emb 512 on a 16-CTA cluster keeps the unit caches in global memory
    cfg, W, obs, noise, ev, d_obs, d_noise = setup("scale256", 2, torch, B, wide_rows=-1)
    S = synth.bernoulli_schedule(36, 100, 0.2, 11)
    got = ev.denoise(d_obs, d_noise, S).cpu().numpy()
    assert ev.last_call()["path"] == "cluster"
    check(got[[1]], oracle_subset(W, cfg, obs, noise, S, [1]), TOL["bf16"], "scale-up cluster")


@pytest.mark.parametrize("n,frac", [(256, 0.125), (1024, 1.0)])
def test_scaleup(torch, B, n, frac):
    name = "scale256" if n == 256 else "scale1024"
    cfg, W, obs, noise, ev, d_obs, d_noise = setup(name, n, torch, B)
    S = synth.bernoulli_schedule(36, 100, frac, 7)
    got = ev.denoise(d_obs, d_noise, S).cpu().numpy()
    assert ev.last_call()["path"] == "wide"
    idx = [0, n - 1]
    check(got[idx], oracle_subset(W, cfg, obs, noise, S, idx), TOL["bf16"], name)


def population_lattices(P: int):
    """P candidate lattices [P][8][100] drawn by Eq. 7 from the synthetic map
    (the oracle's sampler), with budgets of 5-60 % of the cells."""
    d = synth.dissimilarity_map(8, 100, 5)
    Ks = synth.population_budgets(P, 800, 6)
    rnd = synth.guided_randoms(P, int(Ks.max()), 7)
    q = O.guided_weights(d, 0.05, 2)
    return np.stack([O.guided_sample(q, int(Ks[p]), rnd[p]).reshape(8, 100) for p in range(P)])


@pytest.mark.parametrize("path", ["wide", "cluster"])
def test_population_64x16(torch, B, path):
    cfg = synth.config("population")
    W = synth.make_weights(cfg, 0)
    P, N = cfg["n_candidates"], cfg["batch"]
    obs, noise = synth.make_obs(cfg, N, 1), synth.make_noise(cfg, N, 2)
    pop = population_lattices(P)
    # the reference chunks below (N samples) must take the population's path
    ev = B.Evo(cfg, W, (P + 1) * N, wide_rows=N * cfg["horizon"] if path == "wide" else -1)
    x, dev = ev.population(torch.from_numpy(obs).cuda(), torch.from_numpy(noise).cuda(), pop)
    assert ev.last_call()["path"] == path
    x, dev = x.cpu().numpy(), dev.cpu().numpy()
    # deviation is consistent with the returned actions and the all-refresh reference
    full = ev.denoise(torch.from_numpy(obs).cuda(), torch.from_numpy(noise).cuda(),
                      np.ones((24, 100), np.uint8)).cpu().numpy()
    assert ev.last_call()["path"] == path
    host_dev = np.linalg.norm((x - full[None]).reshape(P, N, -1), axis=2).mean(1)
    assert np.allclose(dev, host_dev, rtol=1e-4, atol=1e-5)
    # sampled candidates on every observation against the oracle's population
    # evaluation (its first candidate is the all-refresh lattice, so its actions
    # are the oracle's reference x_full)
    ones = np.ones_like(pop[0])
    sel = [0, 13, P - 1]
    xs_o, dev_o = O.population_deviation(W, cfg, obs, noise, np.stack([ones] + [pop[p] for p in sel]))
    assert dev_o[0] == 0.0
    full_err = np.linalg.norm((full - xs_o[0]).reshape(N, -1), axis=1)
    check(full, xs_o[0], TOL["bf16"], "all-refresh reference")
    for j, p in enumerate(sel):
        check(x[p], xs_o[1 + j], TOL["bf16"], f"candidate {p}")
        # |dev - dev_o| <= mean_n (||x_pn - x_pn^o|| + ||full_n - full_n^o||) by the triangle inequality
        cand_err = np.linalg.norm((x[p] - xs_o[1 + j]).reshape(N, -1), axis=1)
        bound = float(np.mean(cand_err + full_err)) + 1e-5
        assert abs(float(dev[p]) - dev_o[1 + j]) <= bound, (p, dev[p], dev_o[1 + j], bound)
    # denser candidates deviate less on average
    dens = pop.reshape(P, -1).mean(1)
    assert np.corrcoef(dens, dev)[0, 1] < 0
