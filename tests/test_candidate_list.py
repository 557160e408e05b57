"""The selection kernel's incremental candidate list, modelled on the host.

Each CTA of the tensor-core selection keeps a sorted list of up to 64 of its
highest keys w~_i delta_i (lowest index first on ties) and a bound theta that
every other live token's key stays at or below:

  * rebuild: each of the 8 warps ranks the tokens it owns (blocks of 32 at a
    stride of 256) and keeps its 17 best; every token a warp left out has a key at
    or below that warp's 17th, so the union's entries above th = the largest of
    those 17th keys are exactly the CTA's top keys.  The first 64 form the list;
    theta is th, or the 65th such key when more than 64 are above th.
  * refresh (after each update): keys only fall (delta shrinks, w~ >= 0) and
    selected tokens leave, so re-keying the list's own entries and dropping those
    now at or below theta leaves exactly the live tokens above theta.  Fewer than
    17 left (while a bound exists) calls for a rebuild.
  * publish: the list's first 16 entries are the CTA's 16 best keys; the bound
    slot takes the list's 17th entry, or theta when the list holds only 16.  A
    rebuild leaves only 16 when one warp owns the CTA's best 17 keys (its 17th is
    th itself), which happens whenever keys tie and the lowest indices win: equal
    weights on orthogonal features, or weight-zero tokens once the positive ones
    are taken.  Publishing "no bound" there would let a round accept another CTA's
    candidate ahead of this CTA's 17th key.

This file checks those claims against brute force (sorting every live key) over
many rounds of random key decreases and selections, including exact value ties,
tokens of weight zero, and CTAs with fewer live tokens than the published count,
and then runs the batched rounds with this publish against the sequential greedy.
"""
import numpy as np
import pytest

WARPS, TOP, DEEP, PUBLISHED = 8, 17, 64, 17
NONE = (-np.inf, 0)   # below every key


def _key(v, i):
    return (float(v), -int(i))


def _warp_tokens(n, w):
    return [t for t0 in range(w * 32, n, WARPS * 32) for t in range(t0, min(t0 + 32, n))]


def _rebuild(vals, live):
    n = len(vals)
    lists = []
    for w in range(WARPS):
        keys = sorted((_key(vals[t], t) for t in _warp_tokens(n, w) if live[t]), reverse=True)
        lists.append(keys[:TOP] + [NONE] * (TOP - len(keys[:TOP])))
    th = max(lst[TOP - 1] for lst in lists)
    above = sorted((k for lst in lists for k in lst if k > th), reverse=True)
    theta = above[DEEP] if len(above) > DEEP else th
    return above[:DEEP], theta


def _refresh(deep, theta, vals, live):
    kept = []
    for k in deep:
        t = -k[1]
        if live[t]:
            nk = _key(vals[t], t)
            if nk > theta:
                kept.append(nk)
    kept.sort(reverse=True)
    rescan = len(kept) < PUBLISHED and theta != NONE
    return kept, rescan


def _brute(vals, live):
    return sorted((_key(vals[t], t) for t in range(len(vals)) if live[t]), reverse=True)


def _publish(deep, theta, bound_from_theta=True):
    """The 16 candidates and the bound slot a CTA publishes."""
    if len(deep) > PUBLISHED - 1:
        return deep[:PUBLISHED - 1], deep[PUBLISHED - 1]
    return deep, (theta if bound_from_theta else NONE)


@pytest.mark.parametrize("n,seed,ties", [(1366, 1, False), (1366, 2, True), (700, 3, False),
                                         (300, 4, True), (40, 5, False), (12, 6, False)])
def test_incremental_list_holds_the_top_keys(n, seed, ties):
    rng = np.random.default_rng(seed)
    vals = rng.random(n)
    if ties:
        vals = np.round(vals * 8) / 8            # many exact value ties
    vals[rng.random(n) < 0.05] = 0.0             # weight-zero tokens
    live = np.ones(n, bool)
    deep, theta = _rebuild(vals, live)
    rebuilds = 1
    for _ in range(60):
        if not live.any():
            break
        everything = _brute(vals, live)
        # the list is every live key above theta, in order
        assert deep == [k for k in everything if k > theta]
        # publishing: the 16 best, and a bound on every other live key
        cands, bound = _publish(deep, theta)
        assert cands == everything[:len(cands)]
        assert len(cands) == min(PUBLISHED - 1, len(everything))
        if len(everything) > len(cands):
            assert bound >= everything[len(cands)]
        # a round: select a few of the best, lower some keys (never raise one)
        for k in everything[:int(rng.integers(1, 12))]:
            live[-k[1]] = False
        drop = rng.random(n) < 0.3
        vals = np.where(drop, vals * rng.random(n), vals)
        if ties:
            vals = np.floor(vals * 64) / 64
        deep, rescan = _refresh(deep, theta, vals, live)
        if rescan:
            deep, theta = _rebuild(vals, live)
            rebuilds += 1
    assert rebuilds >= 1


def test_rebuild_bound_covers_tokens_outside_the_warp_lists():
    """Every live token outside the rebuilt list has a key at or below theta, even
    when one warp owns all of the highest keys (its 17 best are kept, and the
    others' are dominated by its 17th)."""
    n = 2048
    vals = np.full(n, 0.1)
    own = _warp_tokens(n, 3)
    vals[own] = np.linspace(1.0, 0.5, len(own))
    live = np.ones(n, bool)
    deep, theta = _rebuild(vals, live)
    inside = {-k[1] for k in deep}
    assert all(_key(vals[t], t) <= theta for t in range(n) if t not in inside)
    cands, bound = _publish(deep, theta)
    everything = _brute(vals, live)
    assert cands == everything[:PUBLISHED - 1] and bound >= everything[PUBLISHED - 1]


def test_short_list_after_rebuild_publishes_theta():
    """Equal keys: the lowest indices lead, all owned by warp 0, so the rebuilt list
    holds 16 keys; the bound slot must be theta (the CTA's true 17th key)."""
    vals = np.full(1024, 0.25)
    live = np.ones(1024, bool)
    deep, theta = _rebuild(vals, live)
    assert len(deep) == PUBLISHED - 1
    assert theta == _key(0.25, 16)
    assert _publish(deep, theta)[1] == _brute(vals, live)[PUBLISHED - 1]


def _rounds_with_lists(w, dist, k, C, lcap, bound_from_theta):
    """Batched rounds (see test_batched_acceptance) whose CTAs publish from their
    incremental lists; returns the picks in order."""
    n = len(w)
    bounds = np.linspace(0, n, C + 1).astype(int)
    sel = np.zeros(n, bool)
    seed = -max(_key(w[i], i) for i in range(n))[1]
    seq = [seed]
    sel[seed] = True
    delta = dist[:, seed].copy()

    def local(q):
        lo, hi = bounds[q], bounds[q + 1]
        return w[lo:hi] * delta[lo:hi], ~sel[lo:hi]

    lists = [list(_rebuild(*local(q))) for q in range(C)]
    while len(seq) < k:
        pub, U = [], NONE
        for q in range(C):
            cands, bound = _publish(*lists[q], bound_from_theta)
            pub.extend((c[0], c[1] - bounds[q]) for c in cands)           # global indices
            U = max(U, bound if bound == NONE else (bound[0], bound[1] - bounds[q]))
        above = sorted((c for c in pub if c > U), reverse=True)
        L = [-c[1] for c in above[:lcap]]
        Up = max(U, above[lcap]) if len(above) > lcap else U
        cd = {i: delta[i] for i in L}
        pending, acc = list(L), []
        while pending and len(seq) + len(acc) < k and len(acc) < 32:
            b = max(pending, key=lambda i: _key(w[i] * cd[i], i))
            if not _key(w[b] * cd[b], b) > Up:
                break
            acc.append(b)
            pending.remove(b)
            for i in pending:
                cd[i] = min(cd[i], dist[i, b])
        assert acc
        for b in acc:
            sel[b] = True
            delta = np.minimum(delta, dist[:, b])
        seq.extend(acc)
        for q in range(C):
            kept, rescan = _refresh(lists[q][0], lists[q][1], *local(q))
            lists[q] = list(_rebuild(*local(q))) if rescan else [kept, lists[q][1]]
    return seq


def _tie_cases():
    rng = np.random.default_rng(7)
    yield "orthogonal-equal-w", np.eye(600), np.full(600, 1 / 600)
    x = rng.standard_normal((600, 8))
    w = rng.random(600)
    w[rng.random(600) < 0.7] = 0.0
    yield "zero-w", x, w
    yield "identical", np.ones((600, 8)), np.full(600, 1 / 600)
    yield "clustered", rng.standard_normal((12, 16))[rng.integers(0, 12, 600)], rng.random(600)


@pytest.mark.parametrize("C,lcap", [(2, 16), (2, 32), (5, 32), (16, 32)])
def test_rounds_publishing_from_lists_reproduce_the_greedy(C, lcap):
    from test_batched_acceptance import _cos_dist, _sequential
    for name, x, w in _tie_cases():
        dist = _cos_dist(x)
        want = _sequential(w, dist, 200)
        assert _rounds_with_lists(w, dist, 200, C, lcap, True) == want, name


def test_no_bound_on_a_short_list_breaks_the_rounds():
    """The same rounds with an empty bound slot for a 16-key list pick another CTA's
    candidate ahead of the CTA's 17th key on equal keys (what the theta bound fixes)."""
    from test_batched_acceptance import _cos_dist, _sequential
    x, w = np.eye(600), np.full(600, 1 / 600)
    dist = _cos_dist(x)
    assert _rounds_with_lists(w, dist, 200, 2, 32, False) != _sequential(w, dist, 200)
