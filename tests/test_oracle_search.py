"""Pins of the oracle's schedule search (Sec. 3.2, Sec. 3.3, Eq. 3, 7, 8, 9):
SplitMix64 against its published outputs, the genetic search against brute
force on lattices small enough to enumerate, the invariants every operator
must keep (exactly K unique positions; m per unit in the block-wise variant;
elitism; the signature memo), guided initial individuals against the Eq. 7
sampler, and the early-stopping rule."""
import itertools

import numpy as np
import pytest

from oracle import evo_oracle as O
from oracle.evo_search import Search, SplitMix64


def test_splitmix64_published_outputs():
    r = SplitMix64(0)
    assert [r.next() for _ in range(4)] == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F,
                                            0xF88BB8A8724C81EC]


def _linear(w):
    """fitness = sum of per-cell values of the chosen cells"""
    return lambda S: [float((s.reshape(-1) * w).sum()) for s in S]


def test_finds_brute_force_optimum_on_tiny_lattice():
    U, T, K = 2, 6, 3
    w = np.random.default_rng(0).standard_normal(U * T)
    best = max(sum(w[list(c)]) for c in itertools.combinations(range(U * T), K))
    S, f, st = Search(U, T, K, population=12, elites=4, generations=25, seed=1).run(_linear(w))
    assert f == pytest.approx(best, abs=1e-12)
    assert S.sum() == K


def test_block_wise_finds_brute_force_optimum():
    U, T, m = 3, 5, 2
    w = np.random.default_rng(1).standard_normal(U * T)
    best = sum(np.sort(w[b * T:(b + 1) * T])[-m:].sum() for b in range(U))   # best m per row
    S, f, st = Search(U, T, m, block_wise=True, population=12, elites=4, generations=25, seed=2).run(_linear(w))
    assert f == pytest.approx(best, abs=1e-12)
    assert np.all(S.sum(1) == m)


@pytest.mark.parametrize("block_wise", [False, True])
def test_operators_keep_the_budget_and_memo_avoids_repeats(block_wise):
    U, T = 4, 10
    budget = 3 if block_wise else 12
    seen, per_gen_best = [], []
    w = np.random.default_rng(2).standard_normal(U * T)

    def fit(S):
        for s in S:
            key = tuple(np.flatnonzero(s))
            assert key not in seen                     # the memo never re-evaluates a schedule
            seen.append(key)
            if block_wise:
                assert np.all(s.sum(1) == budget)
            else:
                assert s.sum() == budget
        vals = _linear(w)(S)
        per_gen_best.append(max(vals))
        return vals

    srch = Search(U, T, budget, block_wise=block_wise, population=16, elites=5, generations=12, seed=3)
    S, f, st = srch.run(fit)
    assert st["evaluations"] == len(seen) and st["generations"] == 12
    assert st["evaluations"] + st["memo_hits"] == 16 * 12
    # elitism: the best fitness seen so far never gets lost
    assert f == pytest.approx(max(per_gen_best))


def test_guided_individuals_follow_eq7():
    U, T, K = 4, 25, 20
    d = np.random.default_rng(4).uniform(0.1, 1.0, (U, T)).astype(np.float32)
    calls = []
    srch = Search(U, T, K, population=3, elites=1, generations=1, guided=2, seed=5)
    srch.run(lambda S: (calls.append(S.copy()), [0.0] * len(S))[1], d_map=d)
    # the first guided individual equals the Eq. 7 sampler driven by the same stream
    r = SplitMix64(5)
    rnd = np.array([r.next() for _ in range(K)], dtype=np.uint64)
    want = O.guided_sample(O.guided_weights(d, 0.05, 2), K, rnd).reshape(U, T)
    assert np.array_equal(calls[0][0], want)


def test_early_stopping_accepts_on_formal_score():
    U, T, K = 2, 6, 3
    w = np.arange(U * T, dtype=np.float64)
    best = float(sum(sorted(w)[-K:]))
    target = best - 1.0                                   # reachable
    srch = Search(U, T, K, population=10, elites=3, generations=40, early_stop=True, q_base=target,
                  delta_acc=0.5, seed=6)
    S, f, st = srch.run(_linear(w), formal=lambda S: [v - 0.25 for v in _linear(w)(S)])
    assert st["stopped_early"] == 1 and st["generations"] < 40
    assert f >= target - 0.5                              # Eq. 9 on the formal score
    assert float((S.reshape(-1) * w).sum()) >= target     # Eq. 8 on the quick score
    # an unreachable target never stops early
    srch = Search(U, T, K, population=10, elites=3, generations=5, early_stop=True, q_base=best + 1, seed=6)
    S, f, st = srch.run(_linear(w), formal=_linear(w))
    assert st["stopped_early"] == 0 and st["formal_evaluations"] == 0 and st["generations"] == 5
