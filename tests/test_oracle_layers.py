"""Independent pins for the oracle's denoiser composition (Sec. 3.1: an
L-layer transformer decoder whose layers hold a self-attention, a
cross-attention and an FFN residual branch; the condition tokens feed the
cross-attention).

The oracle writes its layers out by hand (``branch``, ``condition_memory``,
``_embed``, ``_head``).  Here the same weights are loaded into torch.nn
library modules that share nothing with the oracle -- a pre-norm
``TransformerDecoderLayer`` (causal self-attention mask, erf-GELU, eps 1e-5,
no dropout), ``Linear``, ``Mish`` and ``LayerNorm`` -- and run in float64.  The
two must agree to rounding (1e-12).  A mis-wired branch (the FFN normalised
with the cross-attention's LayerNorm, cross-attention keys taken from the
action stream instead of the memory, an output bias added to the wrong
branch, the condition position embedding added after the MLP, a wrong
timestep for the time token, a noise slot off by one) changes the result by
the size of one weight perturbation (about 1e-2) and fails these tests."""
import numpy as np
import pytest

from oracle import evo_oracle as O
from paper_2607_20293_gb300 import synth

torch = pytest.importorskip("torch")

F64 = torch.float64


def _t(x):
    return torch.as_tensor(np.asarray(x, dtype=np.float64))


def _cfg(**over):
    # small shapes with several heads, a horizon that is not a power of two and
    # more than one observation token, so that a transposed operand shows
    c = synth.config("tiny", n_layer=2, n_emb=48, n_head=3, horizon=7, action_dim=3,
                     n_obs=3, obs_dim=11)
    c.update(over)
    return c


def torch_layer(W, cfg, l):
    """torch.nn pre-norm decoder layer holding layer l's weights (the oracle's
    matrices are [in][out]; torch's Linear weights are [out][in])."""
    E, nh, p = cfg["n_emb"], cfg["n_head"], f"l{l}."
    m = torch.nn.TransformerDecoderLayer(
        d_model=E, nhead=nh, dim_feedforward=4 * E, dropout=0.0, activation="gelu",
        layer_norm_eps=O.LN_EPS, batch_first=True, norm_first=True, dtype=F64)
    with torch.no_grad():
        m.norm1.weight.copy_(_t(W[p + "ln1_g"])); m.norm1.bias.copy_(_t(W[p + "ln1_b"]))
        m.norm2.weight.copy_(_t(W[p + "ln2_g"])); m.norm2.bias.copy_(_t(W[p + "ln2_b"]))
        m.norm3.weight.copy_(_t(W[p + "ln3_g"])); m.norm3.bias.copy_(_t(W[p + "ln3_b"]))
        m.self_attn.in_proj_weight.copy_(_t(W[p + "sa_wqkv"]).T)
        m.self_attn.in_proj_bias.copy_(_t(W[p + "sa_bqkv"]))
        m.self_attn.out_proj.weight.copy_(_t(W[p + "sa_wo"]).T)
        m.self_attn.out_proj.bias.copy_(_t(W[p + "sa_bo"]))
        m.multihead_attn.in_proj_weight.copy_(
            torch.cat([_t(W[p + "ca_wq"]).T, _t(W[p + "ca_wkv"]).T], dim=0))
        m.multihead_attn.in_proj_bias.copy_(torch.cat([_t(W[p + "ca_bq"]), _t(W[p + "ca_bkv"])]))
        m.multihead_attn.out_proj.weight.copy_(_t(W[p + "ca_wo"]).T)
        m.multihead_attn.out_proj.bias.copy_(_t(W[p + "ca_bo"]))
        m.linear1.weight.copy_(_t(W[p + "ff_w1"]).T); m.linear1.bias.copy_(_t(W[p + "ff_b1"]))
        m.linear2.weight.copy_(_t(W[p + "ff_w2"]).T); m.linear2.bias.copy_(_t(W[p + "ff_b2"]))
    return m.eval()


def _linear(w, b):
    m = torch.nn.Linear(w.shape[0], w.shape[1], dtype=F64)
    with torch.no_grad():
        m.weight.copy_(_t(w).T)
        m.bias.copy_(_t(b))
    return m


def torch_condition(W, cfg, obs, k):
    """Memory tokens: [time token, obs tokens] + position embedding, then the
    per-token Linear -> Mish -> Linear."""
    N = obs.shape[0]
    obs_emb = _linear(W["obs_w"], W["obs_b"])(_t(obs))
    # the time token is the oracle's sinusoid, pinned on its own values elsewhere
    t_tok = _t(O.time_embedding(k, cfg["n_emb"])).expand(N, 1, -1)
    tok = torch.cat([t_tok, obs_emb], dim=1) + _t(W["cond_pos"])
    mlp = torch.nn.Sequential(_linear(W["cm_w1"], W["cm_b1"]), torch.nn.Mish(),
                              _linear(W["cm_w2"], W["cm_b2"]))
    return mlp(tok)


def torch_eps(W, cfg, x, memory):
    """One denoiser evaluation: input projection + position embedding, the L
    decoder layers, final LayerNorm and output projection."""
    H, E = cfg["horizon"], cfg["n_emb"]
    a = _linear(W["in_w"], W["in_b"])(_t(x)) + _t(W["pos"])
    causal = torch.triu(torch.ones(H, H, dtype=torch.bool), diagonal=1)   # True = masked
    for l in range(cfg["n_layer"]):
        a = torch_layer(W, cfg, l)(a, memory, tgt_mask=causal)
    lnf = torch.nn.LayerNorm(E, eps=O.LN_EPS, dtype=F64)
    with torch.no_grad():
        lnf.weight.copy_(_t(W["lnf_g"])); lnf.bias.copy_(_t(W["lnf_b"]))
    return _linear(W["head_w"], W["head_b"])(lnf(a))


@pytest.mark.parametrize("seed", [0, 1])
def test_decoder_layer_matches_torch(seed):
    cfg = _cfg()
    W = O.as_f64(synth.make_weights(cfg, seed))
    rng = np.random.default_rng(100 + seed)
    N, H, E, C = 3, cfg["horizon"], cfg["n_emb"], 1 + cfg["n_obs"]
    a = rng.standard_normal((N, H, E))
    memory = rng.standard_normal((N, C, E))
    causal = torch.triu(torch.ones(H, H, dtype=torch.bool), diagonal=1)
    with torch.no_grad():
        for l in range(cfg["n_layer"]):
            want = torch_layer(W, cfg, l)(_t(a), _t(memory), tgt_mask=causal).numpy()
            got = a.copy()
            for u in (O.SA, O.CA, O.FFN):
                got = got + O.branch(W, cfg, l, u, got, memory)
            assert np.max(np.abs(got - want)) < 1e-12, f"layer {l}"


def test_each_branch_matches_torch_submodule():
    # the three residual branches one by one: the cached quantity of Eq. 1 is
    # each branch's output, so each must match on its own, not only their sum
    cfg = _cfg()
    W = O.as_f64(synth.make_weights(cfg, 3))
    rng = np.random.default_rng(7)
    N, H, E, C = 2, cfg["horizon"], cfg["n_emb"], 1 + cfg["n_obs"]
    a = _t(rng.standard_normal((N, H, E)))
    mem = _t(rng.standard_normal((N, C, E)))
    causal = torch.triu(torch.ones(H, H, dtype=torch.bool), diagonal=1)
    m = torch_layer(W, cfg, 1)
    with torch.no_grad():
        x = m.norm1(a)
        sa = m.self_attn(x, x, x, attn_mask=causal, need_weights=False)[0]
        ca = m.multihead_attn(m.norm2(a), mem, mem, need_weights=False)[0]
        ff = m.linear2(torch.nn.functional.gelu(m.linear1(m.norm3(a))))
    for u, want in ((O.SA, sa), (O.CA, ca), (O.FFN, ff)):
        got = O.branch(W, cfg, 1, u, a.numpy(), mem.numpy())
        assert np.max(np.abs(got - want.numpy())) < 1e-12, O.UNIT_NAMES[u]


@pytest.mark.parametrize("k", [0, 37, 99])
def test_condition_memory_matches_torch(k):
    cfg = _cfg()
    W = O.as_f64(synth.make_weights(cfg, 2))
    obs = synth.make_obs(cfg, 4, 5)
    with torch.no_grad():
        want = torch_condition(W, cfg, obs, k).numpy()
    got = O.condition_memory(W, cfg, obs, k)
    assert got.shape == (4, 1 + cfg["n_obs"], cfg["n_emb"])
    assert np.max(np.abs(got - want)) < 1e-12


@pytest.mark.parametrize("sampler,n_steps", [("ddim", 10), ("ddpm", 10)])
def test_uncached_loop_matches_torch_denoiser(sampler, n_steps):
    """The whole uncached loop (Sec. 3.1 with every cell refreshed): per step the
    memory for timestep k_t, the torch denoiser's epsilon, then the sampler step
    (pinned on its own against the Gaussian posterior and DDIM's update)."""
    cfg = _cfg(sampler=sampler, n_steps=n_steps)
    W = O.as_f64(synth.make_weights(cfg, 4))
    obs, noise = synth.make_obs(cfg, 2, 8), synth.make_noise(cfg, 2, 9)
    tab = O.sampler_tables(cfg)
    x = noise[0].astype(np.float64)
    with torch.no_grad():
        for t in range(n_steps):
            k = int(tab["timesteps"][t])
            eps = torch_eps(W, cfg, x, torch_condition(W, cfg, obs, k)).numpy()
            z = noise[1 + t].astype(np.float64) if sampler == "ddpm" else None
            x = O.scheduler_step(cfg, tab, x, eps, k, z)
    got = O.denoise_uncached(W, cfg, obs, noise)
    assert np.max(np.abs(got - x)) < 1e-11
    # and the cached loop with the all-refresh lattice is the same computation
    S = np.ones((3 * cfg["n_layer"], n_steps), np.uint8)
    assert np.max(np.abs(O.denoise(W, cfg, obs, noise, S) - x)) < 1e-11
