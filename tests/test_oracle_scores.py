"""Pins for the oracle's scoring (Eq. 6-8, Sec. 3.3), independent of the oracle itself.

Each check below comes from something other than the oracle's own formula:
a hand-worked example, a closed form, a brute-force full P x P causal
attention built with numpy, or an invariant of the definition.
"""
import math
import os

import numpy as np
import pytest

from workloads import custom, f32_to_bf16_bits, bf16_bits_to_f32

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _read_golden(name):
    vals = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            key, *rest = line.split()
            vals[key] = [float(v) for v in rest]
    return vals


def test_hand_worked_three_keys(oracle_mod):
    """Eq. 6-8 by hand: logits ln1, ln2, ln3 -> row (1,2,3)/6 -> w = (1/3, 2/3)."""
    g = _read_golden("scores_three_keys.txt")
    q = np.ones((1, 1, 1, 1), np.float32)
    k = np.array([math.log(v) for v in g["keys_exp"]], np.float32).reshape(1, 3, 1, 1)
    cu = np.array([0, 3], np.int32)
    row = oracle_mod.last_row(q, k, cu, 0, 0, 0, num_kv_heads=1, scale=1.0)
    np.testing.assert_allclose(row, g["row"], rtol=1e-6)
    w = oracle_mod.scores(q, k, cu, [0], [0, 2], num_kv_heads=1, scale=1.0)
    np.testing.assert_allclose(w, g["w"], rtol=1e-6)


def test_equal_keys_give_uniform_weights(oracle_mod):
    """All keys equal -> every attention entry is 1/P -> w_i = 1/N exactly."""
    rng = np.random.default_rng(5)
    B, L, Hq, Hkv, D = 2, 2, 4, 2, 16
    P, N = 11, 7
    q = rng.standard_normal((B, L, Hq, D)).astype(np.float32)
    k = np.broadcast_to(rng.standard_normal(D).astype(np.float32), (L, B * P, Hkv, D)).copy()
    cu = np.array([0, P, 2 * P], np.int32)
    for b in range(B):
        for h in range(Hq):
            row = oracle_mod.last_row(q, k, cu, b, 1, h, num_kv_heads=Hkv)
            np.testing.assert_allclose(row, 1.0 / P, rtol=1e-14)
    w = oracle_mod.scores(q, k, cu, [2, 0], [0, N, 2 * N], num_kv_heads=Hkv)
    np.testing.assert_allclose(w, 1.0 / N, rtol=1e-13)


def _bruteforce_scores(wl):
    """Full causal attention: every position gets a random query row except p*,
    whose query is the workload's q; softmax over the causally masked P x P
    logits; take row P-1, sum the visual columns over layers and heads
    (kv-heads repeated per group), normalise."""
    B, L, Hq, D = wl.q.shape
    Hkv = wl.num_kv_heads
    G = Hq // Hkv
    to64 = (lambda a: bf16_bits_to_f32(a).astype(np.float64)) if wl.dtype == "bf16" else \
        (lambda a: a.astype(np.float64))
    q, k = to64(wl.q), to64(wl.k)
    scale = 1.0 / math.sqrt(D) if wl.scale <= 0 else wl.scale
    rng = np.random.default_rng(123)
    out, rows = [], {}
    for b in range(B):
        s0, s1 = wl.cu_seqlens[b], wl.cu_seqlens[b + 1]
        P = s1 - s0
        v0, N = wl.vis_start[b], wl.cu_vis[b + 1] - wl.cu_vis[b]
        s = np.zeros(N)
        for l in range(L):
            kk = np.repeat(k[l, s0:s1], G, axis=1)          # [P][Hq][D], repeat_kv
            for h in range(Hq):
                Q = rng.standard_normal((P, D))
                Q[P - 1] = q[b, l, h]
                logits = scale * Q @ kk[:, h, :].T
                logits[np.triu_indices(P, 1)] = -np.inf    # causal mask
                A = np.exp(logits - logits.max(axis=1, keepdims=True))
                A /= A.sum(axis=1, keepdims=True)
                rows[(b, l, h)] = A[P - 1]
                s += A[P - 1, v0:v0 + N]
        out.append(s / s.sum())
    return np.concatenate(out), rows


@pytest.mark.parametrize("dtype,Hq,Hkv,L", [("f32", 4, 4, 1), ("bf16", 6, 2, 2), ("bf16", 4, 1, 3)])
def test_bruteforce_full_causal_attention(oracle_mod, dtype, Hq, Hkv, L):
    wl = custom(seed=7, batch=3, n_vis=[5, 9, 3], n_text=[2, 1, 4], n_before=[0, 3, 1],
                num_layers=L, num_q_heads=Hq, num_kv_heads=Hkv, head_dim=8, feat_dim=16,
                dtype=dtype, keep=[1, 2, 1], n_planted=2)
    ref, rows = _bruteforce_scores(wl)
    for (b, l, h), row in rows.items():
        got = oracle_mod.last_row(wl.q, wl.k, wl.cu_seqlens, b, l, h, num_kv_heads=Hkv)
        np.testing.assert_allclose(got, row, rtol=1e-12, atol=1e-15)
    w = oracle_mod.scores(wl.q, wl.k, wl.cu_seqlens, wl.vis_start, wl.cu_vis, num_kv_heads=Hkv)
    np.testing.assert_allclose(w, ref, rtol=1e-12)


def test_rows_sum_to_one_and_weights_normalised(oracle_mod):
    wl = custom(seed=3, batch=2, n_vis=[40, 17], n_text=[9, 30], n_before=[5, 0], num_layers=2,
                num_q_heads=8, num_kv_heads=2, head_dim=32, feat_dim=16, keep=[4, 2])
    for b in range(2):
        for l in range(2):
            for h in range(8):
                row = oracle_mod.last_row(wl.q, wl.k, wl.cu_seqlens, b, l, h, num_kv_heads=2)
                assert abs(row.sum() - 1.0) < 1e-12 and (row > 0).all()
    w = oracle_mod.scores(wl.q, wl.k, wl.cu_seqlens, wl.vis_start, wl.cu_vis, num_kv_heads=2)
    for b in range(2):
        seg = w[wl.cu_vis[b]:wl.cu_vis[b + 1]]
        assert abs(seg.sum() - 1.0) < 1e-12 and (seg > 0).all()


def test_invariances(oracle_mod):
    """Adding one vector to every key of a kv-head shifts that head's logits by a
    constant (softmax unchanged); permuting kv-head groups or layers leaves s unchanged;
    repeating a layer leaves w unchanged (mean over layers == sum after Eq. 8)."""
    rng = np.random.default_rng(11)
    B, L, Hq, Hkv, D, P, N = 1, 2, 6, 3, 16, 23, 12
    q = rng.standard_normal((B, L, Hq, D))
    k = rng.standard_normal((L, P, Hkv, D))
    cu, vs, cv = [0, P], [4], [0, N]
    f = lambda a: np.ascontiguousarray(a, dtype=np.float32)
    base = oracle_mod.scores(f(q), f(k), cu, vs, cv, num_kv_heads=Hkv)
    k2 = k + rng.standard_normal((L, 1, Hkv, D))
    # shift is applied in fp64 before the fp32 cast, so compare loosely
    w2 = oracle_mod.scores(f(q), f(k2), cu, vs, cv, num_kv_heads=Hkv)
    np.testing.assert_allclose(w2, base, rtol=2e-5)
    perm = [2, 0, 1]
    qp = q.reshape(B, L, Hkv, Hq // Hkv, D)[:, :, perm].reshape(B, L, Hq, D)
    kp = k[:, :, perm]
    np.testing.assert_allclose(oracle_mod.scores(f(qp), f(kp), cu, vs, cv, num_kv_heads=Hkv),
                               base, rtol=1e-13)
    np.testing.assert_allclose(
        oracle_mod.scores(f(q[:, ::-1]), f(k[::-1]), cu, vs, cv, num_kv_heads=Hkv), base, rtol=1e-13)
    w1 = oracle_mod.scores(f(q[:, :1]), f(k[:1]), cu, vs, cv, num_kv_heads=Hkv)
    wdup = oracle_mod.scores(f(np.concatenate([q[:, :1]] * 3, axis=1)),
                             f(np.concatenate([k[:1]] * 3, axis=0)), cu, vs, cv, num_kv_heads=Hkv)
    np.testing.assert_allclose(wdup, w1, rtol=1e-13)


def test_text_keys_enter_the_denominator(oracle_mod):
    """Reading: A is the full-row softmax, so a text key that soaks up nearly all of
    head 0's mass leaves w close to head 1's visual softmax alone."""
    rng = np.random.default_rng(2)
    D, N = 4, 6
    P = N + 2
    q = np.zeros((1, 1, 2, D), np.float32)
    q[0, 0, 0, 0] = 1.0
    q[0, 0, 1, 1] = 1.0
    k = np.zeros((1, P, 2, D), np.float32)
    z1 = rng.standard_normal(N).astype(np.float32)
    k[0, :N, 1, 1] = z1                       # head 1 logits over the visual span
    k[0, :N, 0, 0] = rng.standard_normal(N)   # head 0 visual logits ~ N(0,1)
    k[0, N, 0, 0] = 60.0                       # a text key with a dominant logit in head 0
    w = oracle_mod.scores(q, k, [0, P], [0], [0, N], num_kv_heads=2, scale=1.0)
    e = np.exp(z1.astype(np.float64))
    head1_alone = e / e.sum()
    np.testing.assert_allclose(w, head1_alone, rtol=1e-6)


def test_bf16_inputs_are_widened_exactly(oracle_mod):
    """bf16 bit patterns and the same values given as fp32 produce identical scores."""
    wl = custom(seed=9, batch=2, n_vis=[7, 10], n_text=[3, 2], num_layers=1, num_q_heads=4,
                num_kv_heads=2, head_dim=16, feat_dim=16, dtype="bf16", keep=[2, 3])
    a = oracle_mod.scores(wl.q, wl.k, wl.cu_seqlens, wl.vis_start, wl.cu_vis, num_kv_heads=2)
    b = oracle_mod.scores(bf16_bits_to_f32(wl.q), bf16_bits_to_f32(wl.k), wl.cu_seqlens,
                          wl.vis_start, wl.cu_vis, num_kv_heads=2)
    assert np.array_equal(a, b)
    assert np.array_equal(f32_to_bf16_bits(bf16_bits_to_f32(wl.q)), wl.q)


def test_rejects_bad_offsets(oracle_mod):
    q = np.zeros((1, 1, 1, 4), np.float32)
    k = np.zeros((1, 5, 1, 4), np.float32)
    with pytest.raises(ValueError):   # visual span reaches the query position
        oracle_mod.scores(q, k, [0, 5], [1], [0, 4], num_kv_heads=1)
