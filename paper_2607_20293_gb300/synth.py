"""Seeded synthetic inputs for the cached-denoising workloads.

This module only draws random numbers and lays them out; it computes none of
the denoiser, the sampler or the cache rule.  Both the CUDA path (through the
binding) and the CPU oracle (through the tests) take their inputs from here,
so they see identical weights, observations, noise and schedules.

Workload shapes follow the transformer diffusion policy the paper accelerates
(an L-layer decoder with self-attention, cross-attention and FFN residual
branches, Sec. 3.1; 100 denoising steps, Sec. 4.1).  The paper's datasets and
checkpoints are not available, so weights are N(0, 0.02) from a seed and the
observation features are N(0, 1) vectors with the shapes of the paper's
low-dimensional / image-feature conditions.
"""
from __future__ import annotations

import numpy as np

# name -> shape/sampler description.  "n_obs" counts observation tokens; the
# condition memory holds 1 + n_obs tokens (one diffusion-timestep token first).
CONFIGS = {
    "tiny": dict(n_layer=2, n_emb=64, n_head=2, horizon=8, action_dim=2, n_obs=2, obs_dim=20,
                 n_steps=10, sampler="ddim", train_steps=100, dtype="fp32", batch=1),
    "pusht": dict(n_layer=8, n_emb=256, n_head=4, horizon=16, action_dim=2, n_obs=2, obs_dim=20,
                  n_steps=100, sampler="ddpm", train_steps=100, dtype="bf16", batch=1),
    "manip": dict(n_layer=8, n_emb=256, n_head=4, horizon=16, action_dim=10, n_obs=2, obs_dim=256,
                  n_steps=100, sampler="ddpm", train_steps=100, dtype="bf16", batch=64),
    "scale256": dict(n_layer=12, n_emb=512, n_head=8, horizon=32, action_dim=14, n_obs=4, obs_dim=512,
                     n_steps=100, sampler="ddpm", train_steps=100, dtype="bf16", batch=256),
    "scale1024": dict(n_layer=12, n_emb=512, n_head=8, horizon=32, action_dim=14, n_obs=4, obs_dim=512,
                      n_steps=100, sampler="ddpm", train_steps=100, dtype="bf16", batch=1024),
    # 64 candidate schedules x 16 observations on the Push-T-shaped model
    "population": dict(n_layer=8, n_emb=256, n_head=4, horizon=16, action_dim=2, n_obs=2, obs_dim=20,
                       n_steps=100, sampler="ddpm", train_steps=100, dtype="bf16", batch=16,
                       n_candidates=64),
}

WEIGHT_STD = 0.02


def config(name: str, **over) -> dict:
    c = dict(CONFIGS[name])
    c.update(over)
    return c


def n_noise(cfg: dict) -> int:
    """Noise slots: slot 0 is x_T; DDPM draws one more z per loop step."""
    return cfg["n_steps"] + 1 if cfg["sampler"] == "ddpm" else 1


def weight_shapes(cfg: dict) -> list[tuple[str, tuple[int, ...]]]:
    """Ordered (name, shape) list.  Matrices are [in][out] (y = x @ W)."""
    E, A, D, H = cfg["n_emb"], cfg["action_dim"], cfg["obs_dim"], cfg["horizon"]
    C = 1 + cfg["n_obs"]
    out = [("obs_w", (D, E)), ("obs_b", (E,)), ("cond_pos", (C, E)),
           ("cm_w1", (E, 4 * E)), ("cm_b1", (4 * E,)), ("cm_w2", (4 * E, E)), ("cm_b2", (E,)),
           ("in_w", (A, E)), ("in_b", (E,)), ("pos", (H, E))]
    for l in range(cfg["n_layer"]):
        p = f"l{l}."
        out += [(p + "ln1_g", (E,)), (p + "ln1_b", (E,)),
                (p + "sa_wqkv", (E, 3 * E)), (p + "sa_bqkv", (3 * E,)),
                (p + "sa_wo", (E, E)), (p + "sa_bo", (E,)),
                (p + "ln2_g", (E,)), (p + "ln2_b", (E,)),
                (p + "ca_wq", (E, E)), (p + "ca_bq", (E,)),
                (p + "ca_wkv", (E, 2 * E)), (p + "ca_bkv", (2 * E,)),
                (p + "ca_wo", (E, E)), (p + "ca_bo", (E,)),
                (p + "ln3_g", (E,)), (p + "ln3_b", (E,)),
                (p + "ff_w1", (E, 4 * E)), (p + "ff_b1", (4 * E,)),
                (p + "ff_w2", (4 * E, E)), (p + "ff_b2", (E,))]
    out += [("lnf_g", (E,)), ("lnf_b", (E,)), ("head_w", (E, A)), ("head_b", (A,))]
    return out


def _to_bf16_grid(x: np.ndarray) -> np.ndarray:
    """Snap float32 values to the nearest bfloat16 value (ties to even) so that
    both implementations hold bit-identical bf16 parameters."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16 << 16
    return u.astype(np.uint32).view(np.float32)


def make_weights(cfg: dict, seed: int = 0) -> dict[str, np.ndarray]:
    """Weights ~ N(0, 0.02); LayerNorm gains 1 + N(0, 0.02) so that a swapped
    or mis-indexed gain is visible.  bf16 configs get bf16-representable values."""
    rng = np.random.default_rng(seed)
    w = {}
    for name, shape in weight_shapes(cfg):
        v = rng.standard_normal(shape, dtype=np.float64) * WEIGHT_STD
        if name.endswith("_g"):
            v = v + 1.0
        v = v.astype(np.float32)
        if cfg["dtype"] == "bf16":
            v = _to_bf16_grid(v)
        w[name] = v
    return w


def make_obs(cfg: dict, n: int, seed: int = 1) -> np.ndarray:
    rng = np.random.default_rng(seed)
    return rng.standard_normal((n, cfg["n_obs"], cfg["obs_dim"])).astype(np.float32)


def make_noise(cfg: dict, n: int, seed: int = 2) -> np.ndarray:
    """[n_noise][n][H][A]: slot 0 = initial x, slot 1+t = z drawn at loop step t."""
    rng = np.random.default_rng(seed)
    return rng.standard_normal((n_noise(cfg), n, cfg["horizon"], cfg["action_dim"])).astype(np.float32)


def bernoulli_schedule(rows: int, T: int, frac: float, seed: int = 3, force_t0: bool = False) -> np.ndarray:
    """uint8 [rows][T]; each cell refreshed with probability frac."""
    rng = np.random.default_rng(seed)
    s = (rng.random((rows, T)) < frac).astype(np.uint8)
    if force_t0:
        s[:, 0] = 1
    return s


def heterogeneous_schedule(rows: int, T: int, seed: int = 4, lo: float = 0.05, hi: float = 0.6) -> np.ndarray:
    """Each unit row gets its own refresh fraction drawn from U[lo, hi]."""
    rng = np.random.default_rng(seed)
    f = rng.uniform(lo, hi, size=(rows, 1))
    return (rng.random((rows, T)) < f).astype(np.uint8)


def dissimilarity_map(L: int, T: int, seed: int = 5) -> np.ndarray:
    """Synthetic per-block dissimilarity d[l][t] > 0: a smooth random field
    along t times a per-layer level (blocks differ in both pattern and level)."""
    rng = np.random.default_rng(seed)
    t = np.arange(T)
    d = np.empty((L, T))
    for l in range(L):
        field = np.zeros(T)
        for _ in range(4):
            c, w, h = rng.uniform(0, T), rng.uniform(5, 30), rng.uniform(0.2, 1.0)
            field += h * np.exp(-0.5 * ((t - c) / w) ** 2)
        d[l] = (0.05 + field) * rng.uniform(0.2, 1.0)
    return d


def guided_randoms(P: int, K: int, seed: int = 6) -> np.ndarray:
    """Unsigned 64-bit random integers [P][K] for the draws of guided sampling."""
    rng = np.random.default_rng(seed)
    return rng.integers(0, np.iinfo(np.uint64).max, size=(P, K), dtype=np.uint64, endpoint=True)


def population_budgets(P: int, cells: int, seed: int = 6, rho: tuple[float, float] = (0.05, 0.60)) -> np.ndarray:
    """Refresh budgets K_p of P candidates: densities ~ U[rho] of the lattice's cells."""
    rng = np.random.default_rng(seed)
    return np.array([max(1, int(round(rng.uniform(*rho) * cells))) for _ in range(P)])
