"""Pins of the oracle's Top-k selection (Table 5, "LAST (Top-k)"): the k highest
importance scores, ties to the lowest index, reported in descending-score order."""
import itertools

import numpy as np
import pytest


def test_matches_stable_sort(oracle_mod):
    """A library sort is an independent statement of the same selection."""
    rng = np.random.default_rng(3)
    w = rng.dirichlet(np.ones(300)).astype(np.float32)
    w[[7, 40, 41, 299]] = w.max() * 2        # a four-way tie at the top
    w[[100, 101]] = w[50]                    # ties in the middle
    for k in (0, 1, 3, 4, 5, 57, 299, 300):
        expect = np.lexsort((np.arange(len(w)), -w.astype(np.float64)))[:k]
        assert oracle_mod.select_topk(w, k).tolist() == expect.tolist()


def test_negative_zero_ties_positive_zero(oracle_mod):
    w = np.array([0.0, -0.0, 0.5, 0.0, -0.0, 0.25], dtype=np.float32)
    assert oracle_mod.select_topk(w, 6).tolist() == [2, 5, 0, 1, 3, 4]


@pytest.mark.parametrize("seed", range(4))
def test_bruteforce_subsets(oracle_mod, seed):
    """Among all k-subsets, the selected one is the unique subset whose sorted
    (score desc, index asc) key list is lexicographically largest."""
    rng = np.random.default_rng(10 + seed)
    N, k = 9, 4
    w = rng.integers(0, 4, N).astype(np.float32)      # many ties
    def key(sub):
        return sorted(((-float(w[i]), i) for i in sub))
    best = min(itertools.combinations(range(N), k), key=key)
    got = oracle_mod.select_topk(w, k)
    assert sorted(got.tolist()) == list(best)
    # selection order: non-increasing score, ascending index among equals
    for a, b in zip(got[:-1], got[1:]):
        assert w[a] > w[b] or (w[a] == w[b] and a < b)


def test_equals_greedy_on_orthogonal_features(oracle_mod):
    """delta = 1 for every unselected token when features are mutually orthogonal,
    so the importance-weighted greedy of Eq. 9-11 reduces to Top-k."""
    rng = np.random.default_rng(5)
    N, d, k = 40, 64, 17
    x = np.zeros((N, d), np.float32)
    x[np.arange(N), rng.permutation(d)[:N]] = rng.uniform(0.5, 2.0, N).astype(np.float32)
    w = rng.dirichlet(np.ones(N)).astype(np.float32)
    assert oracle_mod.select_topk(w, k).tolist() == oracle_mod.select_fp32(x, w, k).tolist()


def test_uniform_scores_take_first_indices(oracle_mod):
    w = np.full(25, 0.04, np.float32)
    assert oracle_mod.select_topk(w, 7).tolist() == list(range(7))


def test_permutation_equivariance(oracle_mod):
    rng = np.random.default_rng(8)
    N, k = 200, 31
    w = rng.permutation(N).astype(np.float32)          # distinct scores
    perm = rng.permutation(N)
    a = oracle_mod.select_topk(w, k)
    b = oracle_mod.select_topk(w[perm], k)
    assert sorted(perm[b].tolist()) == sorted(a.tolist())


def test_rejects_k_above_n(oracle_mod):
    with pytest.raises(ValueError):
        oracle_mod.select_topk(np.ones(3, np.float32), 4)
