"""CPU oracle for EVO's schedule-driven cached denoising (float64, numpy).

TEST INFRASTRUCTURE ONLY.  Only the tests, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / reference legs of ``bench.py`` may import this module.  The
library path never calls it and shares no code with it; both sides receive
their inputs from the seeded generators in ``paper_2607_20293_gb300.synth``.

What it computes, in the paper's terms:

* The lattice B x T of cacheable units b (self-attention, cross-attention and
  FFN residual branch of each of L decoder layers, B = 3L) and denoising steps
  t in {0..T-1} (Sec. 3.1).
* Cached execution, Eq. 1: at (b, t) in S the branch output r_{b,t} is computed
  and stored in the unit's cache c_b; elsewhere the cached c_b is used.  Caches
  are reset before each action query (Sec. 3.1, Sec. 3.4).
* The fixed-budget schedule S of Eq. 2 and the position-list individual of
  Eq. 3 (loaders below).
* The diffusion sampler around the denoiser, unchanged (Sec. 3.1, Sec. 4.1):
  DDPM with 100 steps, or DDIM (eta = 0) for short loops.

Readings where the paper is silent (each also listed in the design notes):

* Denoiser: pre-norm transformer decoder of the transformer diffusion policy.
  Action tokens a = x W_in + b_in + P_pos; per layer a += SA(LN1 a) (causal),
  a += CA(LN2 a, memory), a += FFN(LN3 a) with erf-GELU, 4E hidden; output
  eps = LN_f(a) W_head + b_head.  LayerNorm eps 1e-5, no dropout.
* Condition memory (1 + n_obs tokens): token 0 = sinusoidal embedding of the
  diffusion timestep k, tokens 1.. = obs W_obs + b_obs; plus a learned
  position embedding, then a per-token MLP E -> 4E (Mish) -> E.  Cross-attention
  sees every memory token (no memory mask).
* "Residual output of unit b" = the branch output including its output bias,
  before it is added to the stream.
* Empty cache: policy "zero" (default) treats a reset cache as a zero tensor,
  so a unit adds nothing until its first refresh and the work is exactly the
  cells of S; policy "force" computes a unit at its first use even when S
  skips it.
* In bf16 mode the cache holds c_b rounded to bfloat16 (round to nearest
  even), because that is the cache's storage type; the refresh itself adds the
  unrounded r_{b,t}.  Everything else is float64 here.
* Sampler: squared-cosine alpha-bar (Nichol & Dhariwal 2021, s = 0.008,
  beta <= 0.999) over 100 training steps, epsilon prediction, x0 clipped to
  [-1, 1].  DDPM uses the "fixed small" posterior variance (Ho et al. 2020)
  with z drawn per step (none at k = 0).  DDIM eta = 0 (Song et al. 2021)
  uses the direction implied by the clipped x0.
* FLOPs: 2 per multiply-accumulate over every matmul (attention QK^T and PV
  counted over the full H x H / H x C score matrix); norms, softmax,
  activations, adds and the sampler are not counted.
"""
from __future__ import annotations

import math

import numpy as np

SA, CA, FFN = 0, 1, 2
UNIT_NAMES = ("SA", "CA", "FFN")
LN_EPS = 1e-5


# --------------------------------------------------------------------------
# lattice and schedule (Sec. 3.1, Eq. 2, Eq. 3)
# --------------------------------------------------------------------------

def expand_schedule(S: np.ndarray, n_layer: int) -> np.ndarray:
    """Canonical unit-level lattice [3L][T].  A layer-level lattice [L][T]
    means that the three units of layer l share row l."""
    S = np.asarray(S)
    if S.ndim != 2:
        raise ValueError("schedule must be 2-D")
    if not np.all((S == 0) | (S == 1)):
        raise ValueError("schedule entries must be 0 or 1")
    if S.shape[0] == 3 * n_layer:
        return S.astype(np.uint8)
    if S.shape[0] == n_layer:
        return np.repeat(S.astype(np.uint8), 3, axis=0)
    raise ValueError("schedule must have L or 3L rows")


def schedule_from_positions(positions, n_units: int, T: int) -> np.ndarray:
    """Individual x = {(b_i, t_i)} (Eq. 3) -> mask; positions must be unique."""
    S = np.zeros((n_units, T), dtype=np.uint8)
    for b, t in positions:
        if not (0 <= b < n_units and 0 <= t < T):
            raise ValueError("position outside the lattice")
        if S[b, t]:
            raise ValueError("duplicate position")
        S[b, t] = 1
    return S


def budget(S: np.ndarray) -> int:
    """|S| = K, the number of refreshed lattice cells (Eq. 2)."""
    return int(np.asarray(S, dtype=np.int64).sum())


# --------------------------------------------------------------------------
# sampler (DDPM / DDIM, unchanged by the method)
# --------------------------------------------------------------------------

def alpha_bar_fn(s: float) -> float:
    return math.cos((s + 0.008) / 1.008 * math.pi / 2) ** 2


def sampler_tables(cfg: dict) -> dict:
    Ttr, T = cfg["train_steps"], cfg["n_steps"]
    betas = np.array([min(1.0 - alpha_bar_fn((i + 1) / Ttr) / alpha_bar_fn(i / Ttr), 0.999)
                      for i in range(Ttr)], dtype=np.float64)
    alphas_cumprod = np.cumprod(1.0 - betas)
    stride = Ttr // T
    timesteps = np.array([(T - 1 - t) * stride for t in range(T)], dtype=np.int64)
    return dict(betas=betas, alphas_cumprod=alphas_cumprod, timesteps=timesteps, stride=stride)


def scheduler_step(cfg: dict, tab: dict, x: np.ndarray, eps: np.ndarray, k: int, z) -> np.ndarray:
    """One reverse step from diffusion timestep k to k - stride."""
    ac = tab["alphas_cumprod"]
    prev = k - tab["stride"]
    ab = ac[k]
    ab_prev = ac[prev] if prev >= 0 else 1.0
    x0 = (x - math.sqrt(1.0 - ab) * eps) / math.sqrt(ab)
    x0 = np.clip(x0, -1.0, 1.0)
    if cfg["sampler"] == "ddpm":
        alpha_t = ab / ab_prev
        beta_t = 1.0 - alpha_t
        mean = (math.sqrt(ab_prev) * beta_t / (1.0 - ab)) * x0 + \
               (math.sqrt(alpha_t) * (1.0 - ab_prev) / (1.0 - ab)) * x
        if k > 0:
            var = max((1.0 - ab_prev) / (1.0 - ab) * beta_t, 1e-20)
            return mean + math.sqrt(var) * z
        return mean
    # DDIM, eta = 0
    eps_dir = (x - math.sqrt(ab) * x0) / math.sqrt(1.0 - ab)
    return math.sqrt(ab_prev) * x0 + math.sqrt(1.0 - ab_prev) * eps_dir


# --------------------------------------------------------------------------
# building blocks
# --------------------------------------------------------------------------

class FlopCounter:
    """Brute-force FLOP count: 2*m*n*k added at every matmul executed."""

    def __init__(self):
        self.total = 0

    def add(self, m: int, n: int, k: int):
        self.total += 2 * m * n * k


def _mm(x: np.ndarray, w: np.ndarray, counter) -> np.ndarray:
    if counter is not None:
        m = int(np.prod(x.shape[:-1]))
        counter.add(m, w.shape[-1], x.shape[-1])
    return x @ w


def layer_norm(x, g, b):
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + LN_EPS) * g + b


def gelu(x):
    from scipy.special import erf
    return 0.5 * x * (1.0 + erf(x / math.sqrt(2.0)))


def mish(x):
    return x * np.tanh(np.logaddexp(0.0, x))


def round_bf16(x: np.ndarray) -> np.ndarray:
    """Round to the nearest bfloat16 value (8 significant bits), ties to even."""
    x = np.asarray(x, dtype=np.float64)
    m, e = np.frexp(x)                      # x = m * 2^e, 0.5 <= |m| < 1
    q = np.ldexp(1.0, e - 8)                # spacing of 8-bit significands in [2^(e-1), 2^e)
    out = np.round(x / q) * q               # np.round: half to even
    return np.where(x == 0, 0.0, out)


def time_embedding(k: int, E: int) -> np.ndarray:
    """Sinusoidal embedding of the diffusion timestep: [sin(k f_i), cos(k f_i)],
    f_i = 10000^(-i/(E/2-1))."""
    half = E // 2
    f = np.exp(-math.log(10000.0) * np.arange(half) / (half - 1))
    return np.concatenate([np.sin(k * f), np.cos(k * f)])


def attention(q, k, v, n_head: int, causal: bool, counter):
    """q [N,Hq,E], k/v [N,Hk,E] -> [N,Hq,E]; softmax(q k^T / sqrt(dh)) v per head."""
    N, Hq, E = q.shape
    Hk = k.shape[1]
    dh = E // n_head
    qh = q.reshape(N, Hq, n_head, dh).transpose(0, 2, 1, 3)
    kh = k.reshape(N, Hk, n_head, dh).transpose(0, 2, 1, 3)
    vh = v.reshape(N, Hk, n_head, dh).transpose(0, 2, 1, 3)
    s = qh @ kh.transpose(0, 1, 3, 2) / math.sqrt(dh)
    if counter is not None:
        counter.add(N * Hq, Hk, E)          # scores, all heads
        counter.add(N * Hq, E, Hk)          # P V, all heads
    if causal:
        mask = np.triu(np.ones((Hq, Hk), dtype=bool), k=1)
        s = np.where(mask, -np.inf, s)
    s = s - s.max(axis=-1, keepdims=True)
    p = np.exp(s)
    p = p / p.sum(axis=-1, keepdims=True)
    o = p @ vh
    return o.transpose(0, 2, 1, 3).reshape(N, Hq, E)


def condition_memory(W, cfg, obs, k, counter=None):
    """Memory tokens [N, 1+n_obs, E] for diffusion timestep k."""
    N = obs.shape[0]
    E = cfg["n_emb"]
    t_tok = np.broadcast_to(time_embedding(k, E), (N, 1, E))
    o_tok = _mm(obs.astype(np.float64), W["obs_w"], counter) + W["obs_b"]
    tok = np.concatenate([t_tok, o_tok], axis=1) + W["cond_pos"]
    h = mish(_mm(tok, W["cm_w1"], counter) + W["cm_b1"])
    return _mm(h, W["cm_w2"], counter) + W["cm_b2"]


def branch(W, cfg, l: int, u: int, a, memory, counter=None):
    """Residual branch output r of unit (layer l, kind u) for stream a."""
    p = f"l{l}."
    E, nh = cfg["n_emb"], cfg["n_head"]
    if u == SA:
        x = layer_norm(a, W[p + "ln1_g"], W[p + "ln1_b"])
        qkv = _mm(x, W[p + "sa_wqkv"], counter) + W[p + "sa_bqkv"]
        q, k, v = qkv[..., :E], qkv[..., E:2 * E], qkv[..., 2 * E:]
        o = attention(q, k, v, nh, True, counter)
        return _mm(o, W[p + "sa_wo"], counter) + W[p + "sa_bo"]
    if u == CA:
        x = layer_norm(a, W[p + "ln2_g"], W[p + "ln2_b"])
        q = _mm(x, W[p + "ca_wq"], counter) + W[p + "ca_bq"]
        kv = _mm(memory, W[p + "ca_wkv"], counter) + W[p + "ca_bkv"]
        o = attention(q, kv[..., :E], kv[..., E:], nh, False, counter)
        return _mm(o, W[p + "ca_wo"], counter) + W[p + "ca_bo"]
    x = layer_norm(a, W[p + "ln3_g"], W[p + "ln3_b"])
    h = gelu(_mm(x, W[p + "ff_w1"], counter) + W[p + "ff_b1"])
    return _mm(h, W[p + "ff_w2"], counter) + W[p + "ff_b2"]


def _embed(W, x, counter):
    return _mm(x, W["in_w"], counter) + W["in_b"] + W["pos"]


def _head(W, a, counter):
    return _mm(layer_norm(a, W["lnf_g"], W["lnf_b"]), W["head_w"], counter) + W["head_b"]


def as_f64(W: dict) -> dict:
    return {k: np.asarray(v, dtype=np.float64) for k, v in W.items()}


# --------------------------------------------------------------------------
# the cached denoising loop (Eq. 1) and the uncached reference loop
# --------------------------------------------------------------------------

def denoise(W, cfg, obs, noise, S, policy: str = "zero", trace=None, counter=None):
    """One action query per sample: noise -> action chunk, following Eq. 1.

    W: weights (float arrays), obs [N][n_obs][D], noise [n_noise][N][H][A],
    S: [3L][T] or [L][T] uint8.  Returns x [N][H][A] (float64).
    trace: optional dict filled with (b, t) -> (refreshed, residual used).
    """
    W = as_f64(W)
    L, T = cfg["n_layer"], cfg["n_steps"]
    U = 3 * L
    S = expand_schedule(S, L)
    if S.shape[1] != T:
        raise ValueError("schedule must have T columns")
    bf16_cache = cfg["dtype"] == "bf16"
    tab = sampler_tables(cfg)
    noise = np.asarray(noise, dtype=np.float64)
    x = noise[0].copy()
    cache = [None] * U                       # reset before the query
    for t in range(T):
        k = int(tab["timesteps"][t])
        memory = condition_memory(W, cfg, obs, k, counter)
        a = _embed(W, x, counter)
        for b in range(U):
            l, u = divmod(b, 3)
            refresh = bool(S[b, t]) or (policy == "force" and cache[b] is None)
            if refresh:
                r = branch(W, cfg, l, u, a, memory, counter)
                cache[b] = round_bf16(r) if bf16_cache else r.copy()
                used = r
            elif cache[b] is not None:
                used = cache[b]
            else:
                used = None                  # reset cache = zero: nothing to add
            if trace is not None:
                trace[(b, t)] = (refresh, None if used is None else used.copy())
            if used is not None:
                a = a + used
        eps = _head(W, a, counter)
        z = noise[1 + t] if cfg["sampler"] == "ddpm" else None
        x = scheduler_step(cfg, tab, x, eps, k, z)
    return x


def denoise_uncached(W, cfg, obs, noise, counter=None):
    """Plain denoiser loop with every branch computed at every step (no cache)."""
    W = as_f64(W)
    tab = sampler_tables(cfg)
    noise = np.asarray(noise, dtype=np.float64)
    x = noise[0].copy()
    for t in range(cfg["n_steps"]):
        k = int(tab["timesteps"][t])
        memory = condition_memory(W, cfg, obs, k, counter)
        a = _embed(W, x, counter)
        for l in range(cfg["n_layer"]):
            for u in (SA, CA, FFN):
                a = a + branch(W, cfg, l, u, a, memory, counter)
        eps = _head(W, a, counter)
        z = noise[1 + t] if cfg["sampler"] == "ddpm" else None
        x = scheduler_step(cfg, tab, x, eps, k, z)
    return x


def population_deviation(W, cfg, obs, noise, S_pop, policy: str = "zero"):
    """Batched candidate evaluation: every schedule S_pop[p] is run on the same
    observations and noise; dev[p] = mean_n || x_p,n - x_full,n ||_2 where
    x_full uses the all-refresh schedule.  Returns (x [P][N][H][A], dev [P])."""
    T, U = cfg["n_steps"], 3 * cfg["n_layer"]
    x_full = denoise(W, cfg, obs, noise, np.ones((U, T), dtype=np.uint8), policy)
    xs, dev = [], []
    for S in S_pop:
        x = denoise(W, cfg, obs, noise, S, policy)
        xs.append(x)
        d = np.sqrt(((x - x_full) ** 2).sum(axis=(1, 2)))
        dev.append(d.mean())
    return np.stack(xs), np.array(dev)


# --------------------------------------------------------------------------
# FLOPs (closed form) -- evo_flops
# --------------------------------------------------------------------------

def unit_flops(cfg: dict) -> tuple[int, int, int]:
    """Per-sample FLOPs of one refresh of an SA, CA and FFN unit."""
    E, H, C = cfg["n_emb"], cfg["horizon"], 1 + cfg["n_obs"]
    sa = 2 * H * E * 3 * E + 2 * H * H * E + 2 * H * H * E + 2 * H * E * E
    ca = 2 * H * E * E + 2 * C * E * 2 * E + 2 * H * C * E + 2 * H * C * E + 2 * H * E * E
    ffn = 2 * H * E * 4 * E + 2 * H * 4 * E * E
    return sa, ca, ffn


def fixed_flops_per_step(cfg: dict) -> int:
    """Per-sample FLOPs every step executes regardless of S: observation
    embedding, condition MLP over all memory tokens, input and output
    projections."""
    E, H, A, D = cfg["n_emb"], cfg["horizon"], cfg["action_dim"], cfg["obs_dim"]
    n_obs = cfg["n_obs"]
    C = 1 + n_obs
    return (2 * n_obs * D * E + 2 * C * E * 4 * E + 2 * C * 4 * E * E
            + 2 * H * A * E + 2 * H * E * A)


def flops_closed_form(cfg: dict, S, policy: str = "zero") -> int:
    S = expand_schedule(S, cfg["n_layer"])
    f = unit_flops(cfg)
    total = cfg["n_steps"] * fixed_flops_per_step(cfg)
    for b in range(S.shape[0]):
        row = S[b]
        n = int(row.sum())
        if policy == "force" and (row.size and row[0] == 0):
            n += 1                           # first use computes the empty unit
        total += n * f[b % 3]
    return total


# ---------------------------------------------------------------------------
# Redundancy-aware initialisation (Sec. 3.3, Eq. 6 and Eq. 7)
# ---------------------------------------------------------------------------
#
# Readings (the paper defines Eq. 6 with the cosine and names, without
# defining them, MSE, L1 and Wasserstein-1 alternatives in its metric
# ablation):
# * a_{r,b,t} is the residual output of unit b at loop step t for sample r of
#   the uncached (all-refresh) policy, flattened over its H x E entries.
# * MSE / L1: the mean over the entries of (a - a')^2 / |a - a'|.
# * Wasserstein-1: between the empirical distributions of the entries of a and
#   a' (equal sample sizes), i.e. the mean of |sort(a) - sort(a')|.
# * Cosine with a zero vector (undefined) counts as dissimilarity 1.
# * "Normalising d into w" is w = d / max d.
# * Eq. 7 draws K distinct positions.  For a result both implementations can
#   reproduce exactly, the weights (eps + w)^gamma are taken in fixed point,
#   q = floor((eps + w)^gamma * 2^40) with gamma a positive integer (repeated
#   products in float64), and draw k picks, among the positions not yet drawn
#   in index order, the first whose running sum of q exceeds rnd_k mod (sum of
#   the remaining q): sequential sampling without replacement with
#   probabilities proportional to q.

METRICS = ("cosine", "mse", "l1", "w1")


def pair_dissimilarity(x, y, metric: str) -> float:
    """The term of Eq. 6 for two activations (cosine: 1 - cos; or a variant)."""
    x = np.asarray(x, dtype=np.float64).ravel()
    y = np.asarray(y, dtype=np.float64).ravel()
    if metric == "cosine":
        nx, ny = np.sqrt(np.dot(x, x)), np.sqrt(np.dot(y, y))
        if nx == 0.0 or ny == 0.0:
            return 1.0
        return 1.0 - float(np.dot(x, y)) / (nx * ny)
    if metric == "mse":
        return float(np.mean((x - y) ** 2))
    if metric == "l1":
        return float(np.mean(np.abs(x - y)))
    if metric == "w1":
        return float(np.mean(np.abs(np.sort(x) - np.sort(y))))
    raise ValueError(metric)


def redundancy_map(acts, metric: str = "cosine"):
    """Eq. 6: acts [R][B][T][...] (activations of R samples) -> d [B][T],
    d_{b,t} = mean over r of 1/(T-1) sum_{t' != t} D(a_{r,b,t}, a_{r,b,t'})."""
    acts = np.asarray(acts)
    R, B, T = acts.shape[:3]
    d = np.zeros((B, T))
    for r in range(R):
        for b in range(B):
            for t in range(T):
                s = 0.0
                for t2 in range(T):
                    if t2 != t:
                        s += pair_dissimilarity(acts[r, b, t], acts[r, b, t2], metric)
                d[b, t] += s / (T - 1)
    return d / R


def trace_activations(trace: dict, U: int, T: int):
    """The denoise trace {(b, t): (refreshed, residual [N][H][E])} of an
    all-refresh query -> activations [N][U][T][H][E]."""
    first = trace[(0, 0)][1]
    N = first.shape[0]
    acts = np.zeros((N, U, T) + first.shape[1:])
    for (b, t), (_, used) in trace.items():
        acts[:, b, t] = used
    return acts


def guided_weights(d, eps: float, gamma: int):
    """Eq. 7 numerators (eps + w)^gamma, w = d / max d, in fixed point (int64,
    2^40 units); eps is taken at float32 precision (the API's argument type)."""
    d = np.asarray(d, dtype=np.float64).ravel()
    w = d / d.max()
    e = np.float64(np.float32(eps))
    q = np.empty(d.size, dtype=np.int64)
    for i in range(d.size):
        base = e + w[i]
        v = base
        for _ in range(gamma - 1):
            v = v * base
        q[i] = int(np.floor(v * 1099511627776.0))
    return q


def guided_sample(q, K: int, rnd):
    """K distinct positions drawn sequentially without replacement with
    probability proportional to q (Eq. 7); rnd [K] unsigned 64-bit integers.
    Draw k: target = rnd_k mod (sum of q over positions not yet drawn); the
    position drawn is the first, in index order, whose running sum of q over
    the positions not yet drawn exceeds the target (when only zero weights
    remain, the first position not yet drawn).  Returns the flat 0/1 lattice."""
    q = np.asarray(q, dtype=np.int64)
    out = np.zeros(q.size, dtype=np.uint8)
    for k in range(K):
        live = np.where(out == 0, q, 0)          # drawn positions add nothing to the running sum
        run = np.cumsum(live)                     # exact: integers
        if run[-1] == 0:                          # only zero weights left: the first position not yet drawn
            out[int(np.flatnonzero(out == 0)[0])] = 1
            continue
        target = int(rnd[k]) % int(run[-1])
        out[int(np.searchsorted(run, target, side="right"))] = 1
    return out


def guided_schedules(d, K: int, eps: float, gamma: int, rnd):
    """P lattices [P][B][T] by Eq. 7 from the map d [B][T]; rnd [P][K]."""
    d = np.asarray(d)
    q = guided_weights(d, eps, gamma)
    return np.stack([guided_sample(q, K, rnd[p]).reshape(d.shape) for p in range(len(rnd))])


# ---------------------------------------------------------------------------
# Baseline schedules (Sec. 1, Sec. 4.1 baselines) and the FLOP table (Table 1)
# ---------------------------------------------------------------------------

def fixed_interval_schedule(B: int, T: int, M: int):
    """EfficientVLA as the paper describes it: every unit refreshed
    synchronously at a fixed temporal interval, M refreshes per unit.  Reading:
    the refresh steps are t_i = floor(i * T / M), i = 0..M-1 (t = 0 included,
    so no unit starts from an empty cache)."""
    S = np.zeros((B, T), dtype=np.uint8)
    for i in range(M):
        S[:, (i * T) // M] = 1
    return S
