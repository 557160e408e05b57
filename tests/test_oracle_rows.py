"""Pins of the oracle's multi-row attention sources (Table 4: First, Middle, All
Mean): the importance of Eq. 7 summed over the causal attention rows of several
query positions, then normalised as in Eq. 8."""
import numpy as np
import pytest

from workloads import bf16_bits_to_f32, f32_to_bf16_bits


def _problem(rng, *, B=2, L=2, Hq=4, Hkv=2, D=16, P=(40, 29), v0=(3, 0), N=(20, 11),
             rows=((25, 31, 39), (11, 28)), dtype="f32"):
    cu_seqlens = np.concatenate([[0], np.cumsum(P)]).astype(np.int32)
    cu_vis = np.concatenate([[0], np.cumsum(N)]).astype(np.int32)
    cu_rows = np.concatenate([[0], np.cumsum([len(r) for r in rows])]).astype(np.int32)
    row_pos = np.array([p for r in rows for p in r], np.int32)
    k = rng.standard_normal((L, int(cu_seqlens[-1]), Hkv, D)).astype(np.float32)
    q = rng.standard_normal((len(row_pos), L, Hq, D)).astype(np.float32)
    if dtype == "bf16":
        k, q = f32_to_bf16_bits(k), f32_to_bf16_bits(q)
    return dict(q=q, k=k, cu_seqlens=cu_seqlens, vis_start=np.array(v0, np.int32),
                cu_vis=cu_vis, cu_rows=cu_rows, row_pos=row_pos, Hkv=Hkv)


def _call(oracle_mod, pr, scale=0.0):
    return oracle_mod.scores_rows(pr["q"], pr["k"], pr["cu_seqlens"], pr["vis_start"],
                                  pr["cu_vis"], pr["cu_rows"], pr["row_pos"],
                                  num_kv_heads=pr["Hkv"], scale=scale)


def _brute_force(pr):
    """Full P x P causal attention per (request, layer, head) in numpy: every
    position gets a query (random where no row sits), the causal mask hides keys
    after each position, and the rows at the requested positions are summed."""
    q, k = pr["q"], pr["k"]
    if q.dtype == np.uint16:
        q, k = bf16_bits_to_f32(q), bf16_bits_to_f32(k)
    q, k = q.astype(np.float64), k.astype(np.float64)
    R, L, Hq, D = q.shape
    Hkv = pr["Hkv"]
    rng = np.random.default_rng(0)
    out = []
    for b in range(len(pr["cu_seqlens"]) - 1):
        s0, s1 = pr["cu_seqlens"][b], pr["cu_seqlens"][b + 1]
        P = s1 - s0
        v0, N = pr["vis_start"][b], pr["cu_vis"][b + 1] - pr["cu_vis"][b]
        rows = range(pr["cu_rows"][b], pr["cu_rows"][b + 1])
        s = np.zeros(N)
        for l in range(L):
            for h in range(Hq):
                g = h // (Hq // Hkv)
                Kb = k[l, s0:s1, g, :]                                   # [P, D]
                Q = rng.standard_normal((P, D))
                for r in rows:                                           # later rows win
                    Q[pr["row_pos"][r]] = q[r, l, h]
                Z = (Q @ Kb.T) / np.sqrt(D)
                Z[np.triu(np.ones((P, P), bool), 1)] = -np.inf           # causal mask
                A = np.exp(Z - Z.max(axis=1, keepdims=True))
                A /= A.sum(axis=1, keepdims=True)
                for r in rows:
                    s += A[pr["row_pos"][r], v0:v0 + N]
        out.append(s / s.sum())
    return np.concatenate(out)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_matches_brute_force_causal_attention(oracle_mod, dtype):
    rng = np.random.default_rng(11)
    # distinct positions per request, so every row is an independent query
    pr = _problem(rng, dtype=dtype)
    np.testing.assert_allclose(_call(oracle_mod, pr), _brute_force(pr), rtol=1e-11, atol=0)


def test_gqa_grouping_and_layers(oracle_mod):
    rng = np.random.default_rng(12)
    pr = _problem(rng, L=3, Hq=6, Hkv=2, D=8, rows=((24, 39), (11, 12, 20, 28)))
    np.testing.assert_allclose(_call(oracle_mod, pr), _brute_force(pr), rtol=1e-11, atol=0)


def test_last_row_alone_is_eq6(oracle_mod):
    """One row at p* = P_b - 1 is the method's own source (Eq. 6-8)."""
    rng = np.random.default_rng(13)
    pr = _problem(rng, rows=((39,), (28,)))
    w_rows = _call(oracle_mod, pr)
    w_last = oracle_mod.scores(pr["q"], pr["k"], pr["cu_seqlens"], pr["vis_start"], pr["cu_vis"],
                               num_kv_heads=pr["Hkv"])
    np.testing.assert_allclose(w_rows, w_last, rtol=1e-13, atol=0)


def test_equal_keys_give_uniform_scores(oracle_mod):
    rng = np.random.default_rng(14)
    pr = _problem(rng)
    pr["k"][:] = pr["k"][:, :1]          # every key equal -> every row uniform
    w = _call(oracle_mod, pr)
    np.testing.assert_allclose(w[:20], np.full(20, 1 / 20), rtol=1e-13)
    np.testing.assert_allclose(w[20:], np.full(11, 1 / 11), rtol=1e-13)


def test_row_order_and_duplicates_do_not_matter(oracle_mod):
    rng = np.random.default_rng(15)
    pr = _problem(rng, rows=((25, 31), (11, 28)))
    base = _call(oracle_mod, pr)
    perm = dict(pr)
    perm["q"] = pr["q"][[1, 0, 3, 2]].copy()
    perm["row_pos"] = pr["row_pos"][[1, 0, 3, 2]].copy()
    np.testing.assert_allclose(_call(oracle_mod, perm), base, rtol=1e-13)
    dup = dict(pr)                        # every row twice: the same normalised scores
    dup["q"] = np.concatenate([pr["q"][:2], pr["q"][:2], pr["q"][2:], pr["q"][2:]])
    dup["row_pos"] = np.concatenate([pr["row_pos"][:2]] * 2 + [pr["row_pos"][2:]] * 2)
    dup["cu_rows"] = np.array([0, 4, 8], np.int32)
    np.testing.assert_allclose(_call(oracle_mod, dup), base, rtol=1e-13)


@pytest.mark.parametrize("bad", [22, 40])   # inside the visual span / past P_b - 1
def test_rejects_rows_outside_the_query(oracle_mod, bad):
    rng = np.random.default_rng(16)
    pr = _problem(rng)
    pr["row_pos"][1] = bad
    with pytest.raises(ValueError):
        _call(oracle_mod, pr)
