"""Pins for the CPU oracle: each test checks it against something other than
itself -- printed values, closed forms, invariants, special cases and brute
force -- so that a dropped term, a wrong sign or index, or a transposed
operand in the oracle fails here."""
import math
import os

import numpy as np
import pytest

from oracle import evo_oracle as O
from paper_2607_20293_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def small_cfg(**over):
    c = synth.config("tiny")
    c.update(over)
    return c


# ---------------------------------------------------------------- primitives

def test_round_bf16_ties_and_values():
    # 1 + 2^-8 lies halfway between 1 and 1 + 2^-7: ties go to the even significand (1).
    assert O.round_bf16(np.array([1 + 2**-8]))[0] == 1.0
    # 1 + 3*2^-8 lies halfway between 1 + 2^-7 (odd) and 1 + 2^-6 (even).
    assert O.round_bf16(np.array([1 + 3 * 2**-8]))[0] == 1 + 2**-6
    assert O.round_bf16(np.array([-(1 + 3 * 2**-8)]))[0] == -(1 + 2**-6)
    # values with 8 significant bits are fixed points
    v = np.array([0.15625, -3.0, 255.0, 2**-20 * 1.5])
    assert np.array_equal(O.round_bf16(v), v)
    assert O.round_bf16(np.array([0.0]))[0] == 0.0
    # relative error bound of 8-bit significands: 2^-9
    x = np.random.default_rng(0).standard_normal(1000)
    assert np.all(np.abs(O.round_bf16(x) - x) <= np.abs(x) * 2**-8)


def test_gelu_pins():
    assert O.gelu(np.array(0.0)) == 0.0
    # Phi(1) from the standard normal table
    assert abs(O.gelu(np.array(1.0)) - 0.8413447460685429) < 1e-15
    # x*Phi(x) - (-x)*Phi(-x) = x for every x
    x = np.linspace(-5, 5, 101)
    assert np.allclose(O.gelu(x) - O.gelu(-x), x, atol=1e-14)


def test_mish_pins():
    assert O.mish(np.array(0.0)) == 0.0
    # tanh(softplus(x)) = ((1+e^x)^2 - 1) / ((1+e^x)^2 + 1)
    for x in (-3.0, -0.5, 1.0, 2.5):
        s = (1 + math.exp(x)) ** 2
        assert abs(O.mish(np.array(x)) - x * (s - 1) / (s + 1)) < 1e-14
    assert abs(O.mish(np.array(30.0)) - 30.0) < 1e-9


def test_layer_norm_invariants():
    rng = np.random.default_rng(1)
    x = rng.standard_normal((5, 64)) * 3 + 2
    y = O.layer_norm(x, np.ones(64), np.zeros(64))
    assert np.allclose(y.mean(-1), 0, atol=1e-12)
    var = x.var(-1)
    assert np.allclose((y ** 2).mean(-1), var / (var + O.LN_EPS), atol=1e-12)
    # constant rows map to beta
    beta = rng.standard_normal(64)
    assert np.allclose(O.layer_norm(np.full((2, 64), 7.0), rng.standard_normal(64), beta), beta)
    # gain and bias act per column
    g = rng.standard_normal(64)
    assert np.allclose(O.layer_norm(x, g, beta), y * g + beta)


def test_time_embedding_pins():
    e0 = O.time_embedding(0, 64)
    assert np.array_equal(e0[:32], np.zeros(32)) and np.array_equal(e0[32:], np.ones(32))
    e = O.time_embedding(7, 64)
    assert abs(e[0] - math.sin(7.0)) < 1e-15 and abs(e[32] - math.cos(7.0)) < 1e-15
    # slowest frequency is 1/10000
    assert abs(e[31] - math.sin(7.0 / 10000.0)) < 1e-15


def test_attention_causal_uniform_is_prefix_mean():
    rng = np.random.default_rng(2)
    N, H, E, nh = 2, 6, 8, 2
    v = rng.standard_normal((N, H, E))
    zeros = np.zeros((N, H, E))
    o = O.attention(zeros, zeros, v, nh, True, None)   # equal scores -> uniform over the allowed keys
    prefix = np.cumsum(v, axis=1) / np.arange(1, H + 1)[None, :, None]
    assert np.allclose(o, prefix, atol=1e-14)
    o_full = O.attention(zeros, zeros, v, nh, False, None)
    assert np.allclose(o_full, v.mean(axis=1, keepdims=True).repeat(H, 1), atol=1e-14)


def test_attention_two_keys_known_weights():
    # one query, two keys; head 0 scores: ln 3 and 0 -> weights 3/4, 1/4
    E, nh, dh = 4, 2, 2
    q = np.zeros((1, 1, E)); k = np.zeros((1, 2, E)); v = np.zeros((1, 2, E))
    q[0, 0, :dh] = [math.log(3.0) * math.sqrt(dh), 0.0]
    k[0, 0, :dh] = [1.0, 0.0]
    v[0, 0, :dh] = [1.0, 2.0]; v[0, 1, :dh] = [5.0, -2.0]
    # head 1: keys scaled so that only key 1 matters
    q[0, 0, dh:] = [0.0, 50.0]; k[0, 1, dh:] = [0.0, 50.0]
    v[0, 0, dh:] = [9.0, 9.0]; v[0, 1, dh:] = [-1.0, 4.0]
    o = O.attention(q, k, v, nh, False, None)[0, 0]
    assert np.allclose(o[:dh], 0.75 * np.array([1.0, 2.0]) + 0.25 * np.array([5.0, -2.0]), atol=1e-14)
    assert np.allclose(o[dh:], [-1.0, 4.0], atol=1e-12)


# ---------------------------------------------------------------- sampler

def test_alpha_bar_table():
    tab = O.sampler_tables(small_cfg(sampler="ddpm", n_steps=100))
    ac, betas = tab["alphas_cumprod"], tab["betas"]
    assert np.all(np.diff(ac) < 0)
    # the product of (1 - beta_i) telescopes to alpha_bar((k+1)/T) / alpha_bar(0) while no beta is clamped
    f = lambda s: math.cos((s + 0.008) / 1.008 * math.pi / 2) ** 2
    for k in (0, 1, 37, 98):
        assert abs(ac[k] - f((k + 1) / 100) / f(0.0)) < 1e-13
    assert betas[-1] == 0.999                       # clamped: alpha_bar(1) = 0
    assert abs(ac[99] - ac[98] * 0.001) < 1e-18
    assert np.array_equal(tab["timesteps"], np.arange(99, -1, -1))
    tab10 = O.sampler_tables(small_cfg())
    assert np.array_equal(tab10["timesteps"], np.arange(90, -1, -10))


def _posterior_by_conditioning(ab_prev, alpha_t, x0, xt):
    # x_{t-1} = sqrt(ab_prev) x0 + sqrt(1-ab_prev) e1 ; x_t = sqrt(alpha_t) x_{t-1} + sqrt(1-alpha_t) e2
    mu1, mu2 = math.sqrt(ab_prev) * x0, math.sqrt(ab_prev * alpha_t) * x0
    s11 = 1 - ab_prev
    s12 = math.sqrt(alpha_t) * (1 - ab_prev)
    s22 = alpha_t * (1 - ab_prev) + (1 - alpha_t)
    return mu1 + s12 / s22 * (xt - mu2), s11 - s12 ** 2 / s22


@pytest.mark.parametrize("k", [1, 10, 50, 98])
def test_ddpm_step_is_gaussian_posterior(k):
    cfg = small_cfg(sampler="ddpm", n_steps=100)
    tab = O.sampler_tables(cfg)
    ac = tab["alphas_cumprod"]
    ab, ab_prev = ac[k], ac[k - 1]
    x0, e = 0.3, -1.1
    xt = math.sqrt(ab) * x0 + math.sqrt(1 - ab) * e
    mean, var = _posterior_by_conditioning(ab_prev, ab / ab_prev, x0, xt)
    # epsilon equal to the true noise recovers x0; z = 0 gives the posterior mean
    got0 = O.scheduler_step(cfg, tab, np.array([xt]), np.array([e]), k, np.array([0.0]))[0]
    got1 = O.scheduler_step(cfg, tab, np.array([xt]), np.array([e]), k, np.array([1.0]))[0]
    assert abs(got0 - mean) < 1e-12
    assert abs((got1 - got0) - math.sqrt(var)) < 1e-12


def test_ddpm_last_step_and_clip():
    cfg = small_cfg(sampler="ddpm", n_steps=100)
    tab = O.sampler_tables(cfg)
    ab = tab["alphas_cumprod"][0]
    # at k = 0 the step returns x0 exactly (alpha_bar_prev = 1) and draws no noise
    x0 = np.array([0.2, -0.7])
    e = np.array([0.5, 1.5])
    x = math.sqrt(ab) * x0 + math.sqrt(1 - ab) * e
    assert np.allclose(O.scheduler_step(cfg, tab, x, e, 0, np.array([9.0, 9.0])), x0, atol=1e-12)
    # a predicted x0 beyond the range is clipped to +-1
    assert np.allclose(O.scheduler_step(cfg, tab, np.array([5.0]), np.array([0.0]), 0, None), [1.0])


def test_ddim_step_eq12():
    cfg = small_cfg()
    tab = O.sampler_tables(cfg)
    ac = tab["alphas_cumprod"]
    k = 50
    x0, e = np.array([0.4]), np.array([0.8])
    x = math.sqrt(ac[k]) * x0 + math.sqrt(1 - ac[k]) * e
    want = math.sqrt(ac[40]) * x0 + math.sqrt(1 - ac[40]) * e
    assert np.allclose(O.scheduler_step(cfg, tab, x, e, k, None), want, atol=1e-12)
    assert np.allclose(O.scheduler_step(cfg, tab, x, e, 0, None),
                       np.clip((x - math.sqrt(1 - ac[0]) * e) / math.sqrt(ac[0]), -1, 1), atol=1e-12)


# ---------------------------------------------------------------- Eq. 1 semantics

def _inputs(cfg, n=2, seed=0):
    W = synth.make_weights(cfg, seed)
    return W, synth.make_obs(cfg, n, seed + 1), synth.make_noise(cfg, n, seed + 2)


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_all_ones_equals_uncached(dtype):
    cfg = small_cfg(dtype=dtype)
    W, obs, noise = _inputs(cfg)
    S = np.ones((3 * cfg["n_layer"], cfg["n_steps"]), np.uint8)
    x1 = O.denoise(W, cfg, obs, noise, S)
    x2 = O.denoise_uncached(W, cfg, obs, noise)
    assert np.array_equal(x1, x2)
    cfg_p = small_cfg(dtype=dtype, sampler="ddpm", n_steps=12, train_steps=12)
    noise_p = synth.make_noise(cfg_p, 2, 5)
    S = np.ones((6, 12), np.uint8)
    assert np.array_equal(O.denoise(W, cfg_p, obs, noise_p, S), O.denoise_uncached(W, cfg_p, obs, noise_p))


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_skipped_cells_return_cached_tensor(dtype):
    cfg = small_cfg(dtype=dtype)
    W, obs, noise = _inputs(cfg)
    S = synth.bernoulli_schedule(6, 10, 0.4, seed=11)
    trace = {}
    O.denoise(W, cfg, obs, noise, S, trace=trace)
    last = {}
    skipped_checked = 0
    for t in range(10):
        for b in range(6):
            refreshed, used = trace[(b, t)]
            assert refreshed == bool(S[b, t])
            if refreshed:
                last[b] = O.round_bf16(used) if dtype == "bf16" else used
            elif b in last:
                assert np.array_equal(used, last[b])
                skipped_checked += 1
            else:
                assert used is None
    assert skipped_checked > 5


def test_all_zero_schedule_is_identity_decoder():
    # under the zero reading, no unit ever adds anything: the decoder is the identity
    cfg = small_cfg()
    W, obs, noise = _inputs(cfg)
    x = O.denoise(W, cfg, obs, noise, np.zeros((6, 10), np.uint8))
    Wd = {k: v.astype(np.float64) for k, v in W.items()}
    ac = O.sampler_tables(cfg)["alphas_cumprod"]
    y = noise[0].astype(np.float64)
    for k in range(90, -1, -10):
        a = np.einsum("nha,ae->nhe", y, Wd["in_w"]) + Wd["in_b"] + Wd["pos"]
        mu = a.mean(-1, keepdims=True)
        sd = np.sqrt(((a - mu) ** 2).mean(-1, keepdims=True) + 1e-5)
        eps = np.einsum("nhe,ea->nha", (a - mu) / sd * Wd["lnf_g"] + Wd["lnf_b"], Wd["head_w"]) + Wd["head_b"]
        ab, abp = ac[k], (ac[k - 10] if k >= 10 else 1.0)
        x0 = np.clip((y - np.sqrt(1 - ab) * eps) / np.sqrt(ab), -1, 1)
        y = np.sqrt(abp) * x0 + np.sqrt(1 - abp) * (y - np.sqrt(ab) * x0) / np.sqrt(1 - ab)
    assert np.allclose(x, y, atol=1e-12)


def test_layer_rows_equal_replicated_unit_rows():
    cfg = small_cfg()
    W, obs, noise = _inputs(cfg)
    SL = synth.bernoulli_schedule(2, 10, 0.5, seed=4)
    SU = np.repeat(SL, 3, axis=0)
    assert np.array_equal(O.denoise(W, cfg, obs, noise, SL), O.denoise(W, cfg, obs, noise, SU))


def test_force_policy_matches_zero_when_t0_refreshes():
    cfg = small_cfg()
    W, obs, noise = _inputs(cfg)
    S = synth.bernoulli_schedule(6, 10, 0.5, seed=7, force_t0=True)
    assert np.array_equal(O.denoise(W, cfg, obs, noise, S, "force"), O.denoise(W, cfg, obs, noise, S, "zero"))
    S[:, 0] = 0
    assert not np.array_equal(O.denoise(W, cfg, obs, noise, S, "force"), O.denoise(W, cfg, obs, noise, S, "zero"))


def test_population_reference_candidate_has_zero_deviation():
    cfg = small_cfg()
    W, obs, noise = _inputs(cfg, n=3)
    pop = np.stack([np.ones((6, 10), np.uint8), synth.bernoulli_schedule(6, 10, 0.3, seed=9)])
    xs, dev = O.population_deviation(W, cfg, obs, noise, pop)
    assert dev[0] == 0.0 and dev[1] > 0
    assert np.isclose(dev[1], np.mean(np.linalg.norm((xs[1] - xs[0]).reshape(3, -1), axis=1)))


# ---------------------------------------------------------------- schedules and FLOPs

def test_positions_roundtrip_and_duplicates():
    S = schedule = O.schedule_from_positions([(0, 3), (5, 9), (2, 0)], 6, 10)
    assert O.budget(S) == 3 and S[5, 9] == 1
    with pytest.raises(ValueError):
        O.schedule_from_positions([(0, 3), (0, 3)], 6, 10)
    with pytest.raises(ValueError):
        O.schedule_from_positions([(6, 0)], 6, 10)
    with pytest.raises(ValueError):
        O.expand_schedule(np.full((6, 10), 2, np.uint8), 2)
    assert schedule is S


@pytest.mark.parametrize("policy", ["zero", "force"])
@pytest.mark.parametrize("seed", [0, 1, 2])
def test_flops_closed_form_equals_counted(policy, seed):
    cfg = small_cfg(n_layer=2, n_emb=32, n_head=2, horizon=5, n_obs=3, obs_dim=7, action_dim=3)
    W = synth.make_weights(cfg, seed)
    obs, noise = synth.make_obs(cfg, 1, seed), synth.make_noise(cfg, 1, seed)
    S = synth.bernoulli_schedule(6, 10, 0.4, seed=seed)
    c = O.FlopCounter()
    O.denoise(W, cfg, obs, noise, S, policy, counter=c)
    assert c.total == O.flops_closed_form(cfg, S, policy)
    c2 = O.FlopCounter()
    O.denoise_uncached(W, cfg, obs, noise, counter=c2)
    assert c2.total == O.flops_closed_form(cfg, np.ones((6, 10), np.uint8))


def test_unit_flops_match_paper_implied_per_step_cost():
    # The paper's FLOP columns: full DP-T 15.77G (Table 1); EfficientVLA, which
    # refreshes every block at M of the 100 steps: 1.64G (M=8), 1.95G (M=10).
    # Both rows give the same per-step cacheable cost (15.77-1.64)/92 = (15.77-1.95)/90.
    implied = (15.77e9 - 1.64e9) / 92
    assert abs(implied - (15.77e9 - 1.95e9) / 90) / implied < 1e-3
    # DP-T shapes: 8 layers, n_emb 256, horizon 10, 1 time + 2 obs condition tokens
    cfg = dict(n_layer=8, n_emb=256, n_head=4, horizon=10, n_obs=2, obs_dim=20, action_dim=10)
    per_step = 8 * sum(O.unit_flops(cfg))
    assert abs(per_step - implied) / implied < 0.005


def _read_golden(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            unit, bac, evo = [p.strip() for p in line.split(";")]
            rows.append((unit, [int(v) for v in bac.split()], [int(v) for v in evo.split()]))
    return rows


@pytest.mark.parametrize("task", ["pusht", "kitchen", "lift_ph"])
def test_published_evo_schedules_have_budget_240(task):
    rows = _read_golden(f"schedules_{task}.txt")
    assert [r[0] for r in rows] == [f"layers.{l}.{u}" for l in range(8) for u in ("SA", "CA", "FFN")]
    pos = [(b, t) for b, (_, _, evo) in enumerate(rows) for t in evo]
    S = O.schedule_from_positions(pos, 24, 100)
    # M = 10 refreshes per unit on average over B = 24 units: K = 240 (Sec. 4.1)
    assert O.budget(S) == 240
    bac = O.schedule_from_positions([(b, t) for b, (_, bl, _) in enumerate(rows) for t in bl], 24, 100)
    assert np.all(bac[:, 0] == 1)          # every BAC row refreshes at the first step


@pytest.mark.parametrize("T,M", [(100, 8), (100, 10), (100, 100), (10, 3), (7, 1)])
def test_fixed_interval_schedule_properties(T, M):
    S = O.fixed_interval_schedule(5, T, M)
    assert np.all(S.sum(1) == M)                       # M refreshes per unit
    assert np.all(S == S[0])                           # all units synchronous
    assert S[0, 0] == 1                                # the first step refreshes
    steps = np.flatnonzero(S[0])
    gaps = np.diff(np.append(steps, T))                # fixed interval: gaps differ by at most one
    assert gaps.max() - gaps.min() <= 1 and gaps.sum() == T
