"""Pins for the oracle's selection, order restore and gather (Eq. 2, 9-12, Sec. 3.2/3.4).

Independent checks: a hand-worked example, brute-force enumeration of greedy
sequences with a materialised N x N cosine-distance matrix of normalised
features (the non-incremental form), special cases with textbook answers
(orthogonal features -> top-k; identical features; uniform weights ->
farthest-point traversal), exact-integer dot products, and rounding-error
bounds for the canonical fp32 dot.
"""
import itertools
import os

import numpy as np
import pytest

from workloads import custom, bf16_bits_to_f32

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _read_golden(name):
    vals = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                key, *rest = line.split()
                vals[key] = [float(v) for v in rest]
    return vals


def test_hand_worked_2d_example(oracle_mod):
    g = _read_golden("select_2d_example.txt")
    x = np.array(g["x"], np.float32).reshape(4, 2)
    w = np.array(g["w"])
    k = int(g["k"][0])
    for sel in (oracle_mod.select_fp32(x, w.astype(np.float32), k), oracle_mod.select_fp64(x, w, k)):
        assert sel.tolist() == [int(v) for v in g["order"]]
        assert oracle_mod.restore_order(sel).tolist() == [int(v) for v in g["sorted"]]


def _greedy_valid(seq, w, dist):
    """Does `seq` satisfy Eq. 9 and Eq. 11 at every step (lowest index on ties), with
    delta recomputed from scratch (Eq. 10) from the materialised distance matrix?"""
    N = len(w)
    if seq[0] != int(np.argmax(w)):
        return False
    for t in range(1, len(seq)):
        chosen = list(seq[:t])
        delta = dist[:, chosen].min(axis=1)
        prod = w * delta
        prod[chosen] = -np.inf
        if seq[t] != int(np.argmax(prod)):      # np.argmax takes the first maximum
            return False
    return True


def _cos_dist(x):
    xb = x / np.linalg.norm(x, axis=1, keepdims=True)
    return 1.0 - xb @ xb.T


@pytest.mark.parametrize("seed", range(6))
def test_bruteforce_enumeration_of_greedy_sequences(oracle_mod, seed):
    rng = np.random.default_rng(seed)
    N, d, k = 7, 5, 4
    x = rng.standard_normal((N, d)).astype(np.float32)
    w = rng.dirichlet(np.ones(N))
    dist = _cos_dist(x.astype(np.float64))
    valid = [s for s in itertools.permutations(range(N), k) if _greedy_valid(s, w, dist)]
    assert len(valid) == 1, "random inputs have a unique greedy sequence"
    assert oracle_mod.select_fp64(x, w, k).tolist() == list(valid[0])
    assert oracle_mod.select_fp32(x, w.astype(np.float32), k).tolist() == list(valid[0])


def test_orthogonal_features_reduce_to_top_k(oracle_mod):
    """Mutually orthogonal features: delta = 1 for every unselected token, so the
    greedy is the (stable) top-k of w (cf. the Top-k variant of Table 5)."""
    rng = np.random.default_rng(1)
    N, d, k = 48, 64, 20
    x = np.zeros((N, d), np.float32)
    x[np.arange(N), rng.permutation(d)[:N]] = rng.uniform(0.5, 3.0, N).astype(np.float32)
    w = rng.dirichlet(np.ones(N)).astype(np.float32)
    w[5] = w[9] = w.max() * 1.5            # an exact tie between two leaders
    expect = np.argsort(-w, kind="stable")[:k]
    assert oracle_mod.select_fp32(x, w, k).tolist() == expect.tolist()
    assert oracle_mod.select_fp64(x, w.astype(np.float64), k).tolist() == expect.tolist()


def test_identical_features_take_lowest_indices(oracle_mod):
    """All features equal (d = 1024, so 1/sqrt(d) is exact and cos = 1 exactly):
    delta = 0 everywhere after the seed, every product ties at 0, and the lowest
    remaining indices are taken in order."""
    N, d, k = 30, 1024, 9
    x = np.ones((N, d), np.float32)
    w = np.random.default_rng(4).dirichlet(np.ones(N)).astype(np.float32)
    j1 = int(np.argmax(w))
    rest = [i for i in range(N) if i != j1][:k - 1]
    assert oracle_mod.select_fp32(x, w, k).tolist() == [j1] + rest
    assert oracle_mod.select_fp64(x, w.astype(np.float64), k).tolist() == [j1] + rest


def _gonzalez(x, k):
    """Textbook farthest-point traversal under cosine distance, started at index 0."""
    dist = _cos_dist(x.astype(np.float64))
    seq = [0]
    while len(seq) < k:
        dmin = dist[:, seq].min(axis=1)
        dmin[seq] = -np.inf
        seq.append(int(np.argmax(dmin)))
    return seq


@pytest.mark.parametrize("seed", range(3))
def test_uniform_weights_give_farthest_point_traversal(oracle_mod, seed):
    rng = np.random.default_rng(100 + seed)
    N, d, k = 64, 32, 16                       # N a power of two: w = 1/N is exact
    x = rng.standard_normal((N, d)).astype(np.float32)
    w = np.full(N, 1.0 / N)
    expect = _gonzalez(x, k)
    assert oracle_mod.select_fp64(x, w, k).tolist() == expect
    assert oracle_mod.select_fp32(x, w.astype(np.float32), k).tolist() == expect


def test_budget_extremes(oracle_mod):
    rng = np.random.default_rng(8)
    N, d = 21, 40
    x = rng.standard_normal((N, d)).astype(np.float32)
    w = rng.dirichlet(np.ones(N)).astype(np.float32)
    assert oracle_mod.select_fp32(x, w, 0).tolist() == []
    assert oracle_mod.select_fp32(x, w, 1).tolist() == [int(np.argmax(w))]
    full = oracle_mod.select_fp32(x, w, N)
    assert sorted(full.tolist()) == list(range(N))
    assert oracle_mod.restore_order(full).tolist() == list(range(N))
    xs = oracle_mod.gather(x, oracle_mod.restore_order(full))
    assert np.array_equal(xs.view(np.uint32), x.view(np.uint32))
    with pytest.raises(ValueError):
        oracle_mod.select_fp32(x, w, N + 1)


def test_zero_norm_feature_has_unit_distance(oracle_mod):
    """Reading: a zero feature has r = 0, so cos = 0 and delta = 1 to every centre."""
    x = np.array([[1, 0], [0, 0], [1, 0.01]], np.float32)
    w = np.array([0.5, 0.2, 0.3], np.float32)
    # after j1 = 0: delta(1) = 1 -> p = 0.2; delta(2) ~ 5e-5 -> p ~ 1.5e-5
    assert oracle_mod.select_fp32(x, w, 2).tolist() == [0, 1]


def test_permutation_equivariance(oracle_mod):
    wl = custom(seed=21, batch=1, n_vis=200, n_text=3, feat_dim=96, dtype="bf16", keep=[40],
                n_clusters=12)
    x = wl.x
    w = np.random.default_rng(3).dirichlet(np.ones(200)).astype(np.float32)
    perm = np.random.default_rng(4).permutation(200)
    base = oracle_mod.select_fp32(x, w, 40)
    permuted = oracle_mod.select_fp32(np.ascontiguousarray(x[perm]), w[perm], 40)
    assert perm[permuted].tolist() == base.tolist()


def test_canonical_agrees_with_fp64_on_separated_data(oracle_mod):
    """Both arithmetic modes make the same decisions unless two candidates are within
    rounding of each other; on clustered data the sequences agree to the end."""
    wl = custom(seed=5, batch=1, n_vis=300, n_text=3, feat_dim=256, dtype="bf16", keep=[60],
                n_clusters=20)
    w = np.random.default_rng(6).dirichlet(np.ones(300) * 0.5)
    a = oracle_mod.select_fp32(wl.x, w.astype(np.float32), 60)
    b = oracle_mod.select_fp64(wl.x, w, 60)
    assert a.tolist() == b.tolist()


def test_canonical_dot_exact_on_integers(oracle_mod):
    """Small integers: every partial sum is exact in fp32, so any summation order
    gives the exact integer dot product -- catches a dropped or repeated term."""
    rng = np.random.default_rng(0)
    for n in (1, 7, 8, 9, 255, 256, 257, 1000, 2048, 2056):
        a = rng.integers(-8, 9, n)
        b = rng.integers(-8, 9, n)
        exact = int(np.dot(a, b))
        for lanes, vec in ((32, 8), (32, 4), (16, 8), (1, 1)):
            got = oracle_mod.dot_canonical(a.astype(np.float32), b.astype(np.float32),
                                           lanes=lanes, vec=vec)
            assert got == exact, (n, lanes, vec)


def test_canonical_dot_error_bound(oracle_mod):
    """|fl(dot) - dot| <= gamma_m * sum |a_i b_i| with m = n/lanes + log2(lanes) + 1
    roundings on any path (Higham, Accuracy and Stability, Sec. 3.1)."""
    rng = np.random.default_rng(1)
    u = 2.0 ** -24
    for n in (100, 1024, 1536, 2048):
        a = rng.standard_normal(n).astype(np.float32)
        b = rng.standard_normal(n).astype(np.float32)
        exact = float(np.dot(a.astype(np.float64), b.astype(np.float64)))
        m = n // 32 + 6
        bound = m * u / (1 - m * u) * float(np.abs(a.astype(np.float64) * b).sum())
        got = oracle_mod.dot_canonical(a, b)
        assert abs(got - exact) <= bound
        assert got == oracle_mod.dot_canonical(b, a)


def test_restore_order_and_gather(oracle_mod):
    rng = np.random.default_rng(2)
    x = rng.standard_normal((50, 24)).astype(np.float32)
    order = rng.permutation(50)[:17].astype(np.int32)
    idx = oracle_mod.restore_order(order)
    assert idx.tolist() == sorted(order.tolist())
    assert np.array_equal(oracle_mod.gather(x, idx), x[np.sort(order)])
    xb = (rng.integers(0, 65535, (50, 24))).astype(np.uint16)
    assert np.array_equal(oracle_mod.gather(xb, idx), xb[np.sort(order)])


@pytest.mark.parametrize("n,num,den,expect", [
    (576, 1, 8, 72), (576, 5, 8, 360), (576, 3, 8, 216), (16384, 1, 20, 820),
    (16384, 1, 8, 2048), (16384, 1, 4, 4096), (257, 1, 8, 33), (0, 1, 8, 0), (7, 1, 1, 7)])
def test_budget_is_ceil_rho_n(oracle_mod, n, num, den, expect):
    assert oracle_mod.budget(n, num, den) == expect


def test_workload_prune_invariants(oracle_mod):
    """Whole path on a small ragged batch: exactly k unique ascending indices per request,
    gathered rows bitwise equal, k = N returns everything."""
    wl = custom(seed=2, batch=4, n_vis=[33, 64, 5, 80], n_text=[3, 9, 1, 4], n_before=[0, 2, 1, 0],
                num_layers=2, num_q_heads=4, num_kv_heads=2, head_dim=32, feat_dim=64,
                keep=[5, 64, 5, 11], n_planted=3)
    out = oracle_mod.prune(wl)
    for b in range(wl.batch):
        k0, k1 = wl.cu_keep[b], wl.cu_keep[b + 1]
        idx = out["idx"][k0:k1]
        n = wl.cu_vis[b + 1] - wl.cu_vis[b]
        assert len(idx) == k1 - k0 and len(set(idx.tolist())) == len(idx)
        assert (np.diff(idx) > 0).all() and idx.min() >= 0 and idx.max() < n
        rows = wl.x[wl.cu_vis[b]:wl.cu_vis[b + 1]][idx]
        assert np.array_equal(out["x_sel"][k0:k1], rows)
    assert out["idx"][wl.cu_keep[1]:wl.cu_keep[2]].tolist() == list(range(64))
    assert bf16_bits_to_f32(wl.x).shape == wl.x.shape
