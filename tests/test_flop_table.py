"""Baseline schedules and the FLOP / Speed x table of the paper (Table 1),
regenerated with the library's FLOP accountant (C ABI, host) at DP-T shapes.

Printed values (Table 1, PH tasks): full 15.77G; EfficientVLA 1.64G (M=8,
9.62x) and 1.95G (M=10, 8.09x); BAC 2.33G / 2.72G; EVO 1.96G / 2.33G.  The
FLOP convention is a reading (2 FLOPs per multiply-accumulate of every matmul,
attention included): it reproduces the full model to 0.2 % and the per-step
cost of the cacheable units to 0.4 % (tests/test_oracle.py); its fixed
per-step part is ~0.8 MFLOP smaller than the paper's implied one, which puts
the fixed-interval rows ~5 % low.  The BAC / EVO rows average task-specific
schedules of which the paper prints three (Appendix tables): for those the
accountant and the oracle agree exactly, and each EVO schedule is cheaper than
BAC's on the same task, as the paper's rows are."""
import ctypes
import os

import numpy as np
import pytest

from oracle import evo_oracle as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
DPT = dict(n_layer=8, n_emb=256, n_head=4, horizon=10, action_dim=10, n_obs=2, obs_dim=20, n_steps=100,
           train_steps=100, sampler="ddpm", dtype="bf16")
FULL_PAPER = 15.77e9


@pytest.fixture(scope="module")
def B():
    from paper_2607_20293_gb300 import binding, build
    build.build()
    binding.load()
    return binding


def _flops(B, S):
    out = ctypes.c_int64()
    S = np.ascontiguousarray(S, dtype=np.uint8)
    rc = B.load().evo_flops_cfg(ctypes.byref(B.make_config(DPT)), S.ctypes.data, S.shape[0], ctypes.byref(out))
    assert rc == B.OK
    return out.value


def _published(task):
    rows = []
    with open(os.path.join(ROOT, "tests", "golden", f"schedules_{task}.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            _, bac, evo = [p.strip() for p in line.split(";")]
            rows.append(([int(v) for v in bac.split()], [int(v) for v in evo.split()]))
    bac = O.schedule_from_positions([(b, t) for b, (bl, _) in enumerate(rows) for t in bl], 24, 100)
    evo = O.schedule_from_positions([(b, t) for b, (_, el) in enumerate(rows) for t in el], 24, 100)
    return bac, evo


@pytest.mark.parametrize("T,M", [(100, 8), (100, 10), (100, 1), (100, 100), (37, 5)])
def test_fixed_interval_generator_matches_oracle(B, T, M):
    assert np.array_equal(B.schedule_fixed_interval(24, T, M), O.fixed_interval_schedule(24, T, M))


def test_fixed_interval_rejects_bad_budget(B):
    out = np.zeros((2, 10), np.uint8)
    assert B.load().evo_schedule_fixed_interval(2, 10, 11, out.ctypes.data) == B.ERR_ARG
    assert B.load().evo_schedule_fixed_interval(2, 10, 0, out.ctypes.data) == B.ERR_ARG


def test_full_model_flops_match_table1(B):
    full = _flops(B, np.ones((24, 100), np.uint8))
    assert full == O.flops_closed_form(DPT, np.ones((24, 100), np.uint8))
    assert abs(full - FULL_PAPER) / FULL_PAPER < 0.005


@pytest.mark.parametrize("M,paper_flops,paper_speed", [(8, 1.64e9, 9.62), (10, 1.95e9, 8.09)])
def test_fixed_interval_rows_of_table1(B, M, paper_flops, paper_speed):
    f = _flops(B, O.fixed_interval_schedule(24, 100, M))
    full = _flops(B, np.ones((24, 100), np.uint8))
    assert abs(f - paper_flops) / paper_flops < 0.06
    assert abs(full / f - paper_speed) / paper_speed < 0.08


@pytest.mark.parametrize("task", ["pusht", "kitchen", "lift_ph"])
def test_published_schedules_flops(B, task):
    bac, evo = _published(task)
    fb, fe = _flops(B, bac), _flops(B, evo)
    assert fb == O.flops_closed_form(DPT, bac) and fe == O.flops_closed_form(DPT, evo)
    assert fe < fb                                   # EVO's schedule is cheaper than BAC's on the same task
    full = _flops(B, np.ones((24, 100), np.uint8))
    # within the range the paper's rows span (EVO 8.05x..6.77x, BAC 6.77x..5.80x), with the convention's margin
    assert 5.5 < full / fb < 7.5 and 6.5 < full / fe < 9.0
