"""Host-side checks of the C ABI (no GPU needed): the library loads and exports
every entry point declared in include/evo.h; the host entry points (weight
count, FLOP accountant, position-list loader) agree bit-exactly with the oracle."""
import ctypes
import os
import re

import numpy as np
import pytest

from oracle import evo_oracle as O
from paper_2607_20293_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "evo.h")


@pytest.fixture(scope="module")
def B():
    from paper_2607_20293_gb300 import binding, build
    build.build()
    binding.load()
    return binding


def declared_symbols():
    txt = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:evo_status|size_t|const char\*)\s+(evo_\w+)\s*\(", txt, re.M)))


def test_exports_every_declared_symbol(B):
    syms = declared_symbols()
    assert len(syms) >= 11
    lib = ctypes.CDLL(B.LIB_PATH)
    for s in syms:
        assert hasattr(lib, s), s


def test_status_strings(B):
    assert B.status_string(0) == "ok"
    assert "schedule" in B.status_string(3)


@pytest.mark.parametrize("name", list(synth.CONFIGS))
def test_weight_count_matches_generator(B, name):
    cfg = synth.config(name)
    n = sum(int(np.prod(s)) for _, s in synth.weight_shapes(cfg))
    assert B.load().evo_weight_count(ctypes.byref(B.make_config(cfg))) == n
    assert [k for k, _ in synth.weight_shapes(cfg)] == B.weight_names(cfg)


def test_invalid_config_rejected(B):
    cfg = synth.config("tiny", n_head=3)
    assert B.load().evo_weight_count(ctypes.byref(B.make_config(cfg))) == 0


@pytest.mark.parametrize("name", ["tiny", "pusht", "scale256"])
@pytest.mark.parametrize("policy", ["zero", "force"])
def test_flops_bit_exact_vs_oracle(B, name, policy):
    cfg = synth.config(name)
    L, T = cfg["n_layer"], cfg["n_steps"]
    for seed, frac in [(0, 0.5), (1, 0.125), (2, 1.0), (3, 0.0)]:
        S = synth.bernoulli_schedule(3 * L, T, frac, seed)
        assert B.flops_cfg(cfg, S, policy) == O.flops_closed_form(cfg, S, policy)
        SL = synth.bernoulli_schedule(L, T, frac, seed + 10)
        assert B.flops_cfg(cfg, SL, policy) == O.flops_closed_form(cfg, SL, policy)


def test_flops_rejects_bad_lattice(B):
    cfg = synth.config("tiny")
    S = np.zeros((6, 10), np.uint8)
    S[2, 3] = 2
    with pytest.raises(B.EvoError) as e:
        B.flops_cfg(cfg, S)
    assert e.value.code == B.ERR_SCHEDULE
    with pytest.raises(B.EvoError):
        B.flops_cfg(cfg, np.zeros((5, 10), np.uint8))


def _golden_positions(task):
    pos = []
    with open(os.path.join(ROOT, "tests", "golden", f"schedules_{task}.txt")) as f:
        rows = [l for l in f if l.strip() and not l.startswith("#")]
    for b, line in enumerate(rows):
        evo = line.split(";")[2].split()
        pos += [(b, int(t)) for t in evo]
    return pos


@pytest.mark.parametrize("task", ["pusht", "kitchen", "lift_ph"])
def test_positions_loader_bit_exact(B, task):
    pos = _golden_positions(task)
    S = B.schedule_from_positions(pos, 24, 100)
    assert np.array_equal(S, O.schedule_from_positions(pos, 24, 100))
    assert int(S.sum()) == 240
    cfg = synth.config("pusht")
    assert B.flops_cfg(cfg, S) == O.flops_closed_form(cfg, S)


def test_positions_loader_rejects(B):
    with pytest.raises(B.EvoError):
        B.schedule_from_positions([(0, 1), (0, 1)], 6, 10)
    with pytest.raises(B.EvoError):
        B.schedule_from_positions([(6, 1)], 6, 10)
    with pytest.raises(B.EvoError):
        B.schedule_from_positions([(0, 10)], 6, 10)
    assert B.schedule_from_positions([], 6, 10).sum() == 0


def test_argument_checks_before_any_device_work(B):
    # rejected on the host, before the CUDA runtime is touched
    lib = B.load()
    assert lib.evo_test_gelu(None, None, -1, 0, None) == B.ERR_ARG
    assert lib.evo_test_gelu(None, None, 4, 0, None) == B.ERR_ARG
    assert lib.evo_test_gelu(None, None, 0, 2, None) == B.ERR_ARG
    assert lib.evo_test_wait_timeout(None, 0, 100, None) == B.ERR_ARG


def test_binding_rejects_non_contiguous_buffers(B):
    a = np.zeros((4, 6), np.float32)
    with pytest.raises(ValueError):
        B._ptr(a[:, ::2])
    assert B._ptr(a) == a.ctypes.data
    assert B._ptr(None) is None
    torch = pytest.importorskip("torch")
    t = torch.zeros(4, 6)
    with pytest.raises(ValueError):
        B._ptr(t.t())
    assert B._ptr(t) == t.data_ptr()
