"""The library's schedule search (evo_search, host C++) against the oracle
search on the same deterministic fitness: identical best schedule, fitness
and statistics (every random choice comes from the same SplitMix64 stream;
decisions compare identical fitness values).  CPU only."""
import numpy as np
import pytest

from oracle import evo_oracle as O
from oracle.evo_search import Search


@pytest.fixture(scope="module")
def B():
    from paper_2607_20293_gb300 import binding, build
    build.build()
    binding.load()
    return binding


def _linear(w):
    return lambda S: [float((s.reshape(-1) * w).sum()) for s in S]


def _quadratic(w, pairs):
    """a non-additive fitness: cell values plus pair bonuses"""
    def f(S):
        out = []
        for s in S:
            x = s.reshape(-1).astype(np.float64)
            out.append(float(x @ w + sum(v * x[i] * x[j] for i, j, v in pairs)))
        return out
    return f


CASES = [
    dict(U=6, T=20, budget=15, population=12, elites=4, generations=8, seed=1),
    dict(U=6, T=20, budget=2, block_wise=True, population=12, elites=3, generations=8, seed=2),
    dict(U=8, T=25, budget=30, population=16, elites=5, generations=6, guided=6, seed=3),
    dict(U=5, T=12, budget=2, block_wise=True, population=10, elites=2, generations=6, guided=4, seed=4,
         crossover_rate=0.5, mutation_rate=0.1, tournament=2),
]


@pytest.mark.parametrize("case", range(len(CASES)))
@pytest.mark.parametrize("fitness", ["linear", "quadratic"])
def test_search_matches_oracle(B, case, fitness):
    kw = dict(CASES[case])
    U, T = kw.pop("U"), kw.pop("T")
    rng = np.random.default_rng(10 + case)
    w = rng.standard_normal(U * T)
    pairs = [(int(i), int(j), float(v)) for i, j, v in zip(rng.integers(0, U * T, 20), rng.integers(0, U * T, 20),
                                                            rng.standard_normal(20))]
    f = _linear(w) if fitness == "linear" else _quadratic(w, pairs)
    d = rng.uniform(0.05, 1.0, (U, T)).astype(np.float32)
    budget = kw.pop("budget")
    want_S, want_f, want_st = Search(U, T, budget, **kw).run(f, d_map=d)
    got_S, got_f, got_st = B.search(U, T, budget, f, d_map=d, **kw)
    assert np.array_equal(got_S, want_S)
    assert got_f == want_f
    assert got_st == want_st


def test_search_early_stopping_matches_oracle(B):
    U, T, K = 4, 10, 6
    w = np.random.default_rng(20).standard_normal(U * T)
    best = float(np.sort(w)[-K:].sum())
    kw = dict(population=10, elites=3, generations=30, early_stop=True, q_base=best - 2.5, delta_acc=0.2, seed=7)
    formal = lambda S: [v - 0.1 for v in _linear(w)(S)]
    want = Search(U, T, K, **kw).run(_linear(w), formal=formal)
    got = B.search(U, T, K, _linear(w), formal=formal, **kw)
    assert np.array_equal(got[0], want[0]) and got[1] == want[1] and got[2] == want[2]
    assert got[2]["stopped_early"] == 1


def test_search_argument_errors(B):
    with pytest.raises(B.EvoError):
        B.search(4, 10, 50, _linear(np.ones(40)))                      # budget above the lattice
    with pytest.raises(B.EvoError):
        B.search(4, 10, 5, _linear(np.ones(40)), guided=2)             # guided individuals need a map
    with pytest.raises(B.EvoError):
        B.search(4, 10, 5, _linear(np.ones(40)), early_stop=True)      # early stopping needs a formal fitness


def test_fitness_errors_propagate(B):
    def bad(S):
        raise ValueError("fitness failed")
    with pytest.raises(ValueError):
        B.search(4, 10, 5, bad)
