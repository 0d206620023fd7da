"""Pins of the oracle's redundancy-aware initialisation: the dissimilarity map
of Eq. 6 (cosine) and its MSE / L1 / Wasserstein-1 variants, and guided
sampling (Eq. 7).  Hand-computed cases, a library routine for Wasserstein-1,
invariants, and sampling frequencies against closed-form probabilities."""
import numpy as np
import pytest

from oracle import evo_oracle as O


def _acts(rows):
    """one sample, one unit, T = len(rows) activations"""
    return np.asarray(rows, dtype=np.float64)[None, None]


def test_cosine_hand_example():
    # a0 and a1 point the same way, a2 is orthogonal to both
    d = O.redundancy_map(_acts([[1, 0], [2, 0], [0, 1]]), "cosine")
    assert np.allclose(d, [[0.5, 0.5, 1.0]], atol=1e-15)


def test_cosine_is_scale_invariant_and_averages_over_samples():
    rng = np.random.default_rng(0)
    a = rng.standard_normal((2, 3, 5, 4, 6))
    d = O.redundancy_map(a, "cosine")
    scale = rng.uniform(0.1, 10.0, size=(2, 3, 5, 1, 1))
    assert np.allclose(O.redundancy_map(a * scale, "cosine"), d, atol=1e-12)
    d0, d1 = O.redundancy_map(a[:1], "cosine"), O.redundancy_map(a[1:], "cosine")
    assert np.allclose(d, 0.5 * (d0 + d1), atol=1e-14)
    assert np.all(d >= 0) and np.all(d <= 2)


def test_cosine_zero_vector_counts_as_dissimilar():
    d = O.redundancy_map(_acts([[0, 0], [1, 0]]), "cosine")
    assert np.allclose(d, [[1.0, 1.0]])


def test_mse_and_l1_hand_examples():
    a = _acts([[0, 0], [1, 1], [2, 0]])
    # mse: (0,1) -> 1, (0,2) -> 2, (1,2) -> 1 ; l1: every pair -> 1
    assert np.allclose(O.redundancy_map(a, "mse"), [[1.5, 1.0, 1.5]], atol=1e-15)
    assert np.allclose(O.redundancy_map(a, "l1"), [[1.0, 1.0, 1.0]], atol=1e-15)


def test_w1_matches_scipy_and_ignores_order():
    scipy_stats = pytest.importorskip("scipy.stats")
    rng = np.random.default_rng(1)
    for _ in range(5):
        x, y = rng.standard_normal(64), rng.standard_normal(64) * 2 + 0.5
        assert O.pair_dissimilarity(x, y, "w1") == pytest.approx(scipy_stats.wasserstein_distance(x, y), rel=1e-12)
        assert O.pair_dissimilarity(x, y, "w1") <= O.pair_dissimilarity(x, y, "l1") + 1e-15
    x = rng.standard_normal(32)
    assert O.pair_dissimilarity(x, rng.permutation(x), "w1") == 0.0


def test_trace_activations_layout():
    rng = np.random.default_rng(2)
    tr = {(b, t): (True, rng.standard_normal((3, 4, 5))) for b in range(2) for t in range(6)}
    a = O.trace_activations(tr, 2, 6)
    assert a.shape == (3, 2, 6, 4, 5)
    assert np.array_equal(a[1, 1, 4], tr[(1, 4)][1][1])


def test_guided_weights_fixed_point():
    # gamma 1, eps 0: q = w * 2^40 exactly for dyadic w
    assert list(O.guided_weights(np.array([1.0, 2.0, 4.0]), 0.0, 1)) == [2 ** 38, 2 ** 39, 2 ** 40]
    q = O.guided_weights(np.array([1.0, 3.0]), 0.05, 2)
    e = float(np.float32(0.05))
    assert q[1] == int(np.floor((e + 1.0) ** 2 * 2 ** 40))


def test_guided_sample_degenerate_cases():
    q = np.ones(6, dtype=np.int64)
    assert list(O.guided_sample(q, 6, np.arange(6, dtype=np.uint64))) == [1] * 6
    # target 0 takes the first position not yet drawn
    assert list(O.guided_sample(q, 3, np.zeros(3, dtype=np.uint64))) == [1, 1, 1, 0, 0, 0]


def test_guided_sample_frequencies_match_eq7():
    rng = np.random.default_rng(3)
    q = np.array([1, 2, 3, 4], dtype=np.int64) << 20
    p = q / q.sum()
    n = 20000
    rnd = rng.integers(0, 2 ** 63, size=(n, 2), dtype=np.uint64)
    first = np.array([np.argmax(O.guided_sample(q, 1, r)) for r in rnd[:, :1]])
    assert np.allclose(np.bincount(first, minlength=4) / n, p, atol=0.015)
    # K = 2: P({i, j}) = p_i p_j / (1 - p_i) + p_j p_i / (1 - p_j)
    pairs = {}
    for r in rnd[:5000]:
        s = tuple(np.flatnonzero(O.guided_sample(q, 2, r)))
        pairs[s] = pairs.get(s, 0) + 1
    for (i, j), c in pairs.items():
        want = p[i] * p[j] / (1 - p[i]) + p[j] * p[i] / (1 - p[j])
        assert abs(c / 5000 - want) < 0.03
