"""Pins of the oracle's keep-set selection and compaction (Algorithm
DoMemRefresh) by brute force and invariants (no GPU)."""
import numpy as np
import pytest

import oracle


def brute_keep(scores, n, budget, n_sink):
    """Python sort of (score, slot) descending; NaN -> -inf; sinks -> +inf."""
    items = []
    for j in range(n):
        s = float(scores[j])
        if s != s:
            s = float("-inf")
        if j < n_sink:
            s = float("inf")
        items.append((s, j))
    items.sort(reverse=True)
    return sorted(j for _, j in items[:min(budget, n)])


@pytest.mark.parametrize("seed", range(6))
def test_select_matches_brute_force_with_ties(seed):
    r = np.random.default_rng(seed)
    b, cap = 3, 40
    scores = r.integers(-3, 4, size=(b, cap)).astype(np.float32)   # many ties
    scores[0, 5] = np.nan
    scores[1, 7] = np.inf
    scores[2, 0] = -np.inf
    lens = [40, 17, 1]
    budget = [11, 17, 1]
    n_sink = seed % 3
    idx, cnt = oracle.select_keep(scores, lens, budget, n_sink)
    for bi in range(b):
        want = brute_keep(scores[bi], lens[bi], budget[bi], n_sink)
        assert cnt[bi] == len(want)
        assert idx[bi, :cnt[bi]].tolist() == want
        assert np.all(idx[bi, cnt[bi]:] == -1)


def test_select_identity_when_budget_covers_sequence():
    s = np.random.default_rng(1).normal(size=(2, 9)).astype(np.float32)
    idx, cnt = oracle.select_keep(s, [9, 5], [9, 100], 0)
    assert cnt.tolist() == [9, 5]
    assert idx[0].tolist() == list(range(9)) and idx[1, :5].tolist() == list(range(5))


def test_select_ties_prefer_later_slot_and_keep_sinks():
    s = np.zeros((1, 8), np.float32)
    idx, cnt = oracle.select_keep(s, [8], [3], n_sink=0)
    assert idx[0, :3].tolist() == [5, 6, 7]
    idx, cnt = oracle.select_keep(s, [8], [3], n_sink=2)
    assert idx[0, :3].tolist() == [0, 1, 7]


def test_select_signed_zeros_tie_to_the_later_slot():
    # -0.0 == +0.0 as floats: a score -logit of an exactly-zero logit is -0.0
    # and ties with +0.0; the later slot wins whatever the signs
    s = np.array([[0.0, -0.0, -1.0]], np.float32)
    idx, cnt = oracle.select_keep(s, [3], [1])
    assert idx[0, :1].tolist() == [1]
    s = np.array([[-0.0, 0.0, -1.0]], np.float32)
    idx, cnt = oracle.select_keep(s, [3], [1])
    assert idx[0, :1].tolist() == [1]
    r = np.random.default_rng(5)
    for _ in range(20):
        s = np.where(r.random(50) < 0.5, np.float32(-0.0), np.float32(0.0)).astype(np.float32)
        s[r.integers(0, 50, 5)] = r.choice([np.nan, 1.0, -1.0], 5)
        budget = int(r.integers(1, 50))
        idx, cnt = oracle.select_keep(s[None], [50], [budget])
        assert idx[0, :cnt[0]].tolist() == brute_keep(s, 50, budget, 0)


def test_select_keeps_highest_exactly():
    s = np.array([[0.5, 3.0, -1.0, 2.0, 2.5, -7.0]], np.float32)
    idx, cnt = oracle.select_keep(s, [6], [3])
    assert idx[0, :3].tolist() == [1, 3, 4]


def sequential_compact(buf, keep_idx, keep_count):
    """The ascending in-place loop: dst[k] = src[keep_idx[k]] one slot at a time.
    Safe in place because keep_idx is ascending, so keep_idx[k] >= k."""
    out = buf.copy()
    for b in range(buf.shape[0]):
        for k in range(int(keep_count[b])):
            out[b, k] = out[b, keep_idx[b, k]]
    return out


@pytest.mark.parametrize("kind", ["shift1", "all", "last", "random", "sparse_tail", "empty"])
def test_compact_matches_sequential_in_place_loop(kind):
    r = np.random.default_rng(3)
    b, cap = 2, 64
    buf = r.integers(0, 1 << 30, size=(b, cap, 3)).astype(np.int64)
    idx = np.full((b, cap), -1, np.int32)
    cnt = np.zeros(b, np.int32)
    for bi in range(b):
        n = cap - 7 * bi
        if kind == "shift1":
            k = list(range(1, n))
        elif kind == "all":
            k = list(range(n))
        elif kind == "last":
            k = [n - 1]
        elif kind == "random":
            k = sorted(r.choice(n, size=n // 3, replace=False).tolist())
        elif kind == "sparse_tail":
            k = list(range(n - 5, n))
        else:
            k = []
        idx[bi, :len(k)] = k
        cnt[bi] = len(k)
    got = oracle.compact(buf, idx, cnt)
    np.testing.assert_array_equal(got, sequential_compact(buf, idx, cnt))
    for bi in range(b):
        kept = got[bi, :cnt[bi]]
        np.testing.assert_array_equal(kept, buf[bi, idx[bi, :cnt[bi]]])
        np.testing.assert_array_equal(got[bi, cnt[bi]:], buf[bi, cnt[bi]:])


def test_compact_preserves_relative_order():
    buf = np.arange(20)[None, :, None]          # slot value == original slot
    idx = np.array([[2, 3, 9, 11, 19] + [-1] * 15], np.int32)
    out = oracle.compact(buf, idx, np.array([5]))
    assert out[0, :5, 0].tolist() == [2, 3, 9, 11, 19]
    assert np.all(np.diff(out[0, :5, 0]) > 0)


def test_keep_set_bar_accepts_only_near_tie_swaps():
    """The GPU tests' keep-set bar: swaps at a near-tied boundary pass while
    the overlap stays >= 99.5 %, a third swap (overlap 99.25 % at J = 400)
    fails, a swap of a slot far from the boundary fails, a count mismatch
    fails, and at J < 200 a single near-tie swap already fails."""
    from tests._util import keep_set_ok
    n, j = 1000, 400
    s = np.linspace(10.0, -10.0, n)
    s[j - 3:j + 3] = s[j - 1] - 1e-4 * np.arange(6)   # six near-tied slots at the boundary
    want_i, want_c = oracle.select_keep(s[None].astype(np.float32), [n], [j])
    kept = list(want_i[0, :j])

    def swap(k):   # drop the k lowest kept, take the k highest dropped
        return sorted(set(kept) - set(range(j - k, j)) | set(range(j, j + k)))
    far = sorted(set(kept) - {0} | {n - 1})    # drop the best, keep the worst
    for got, expect in ((kept, True), (swap(1), True), (swap(2), True), (swap(3), False),
                        (far, False)):
        gi = np.full((1, n), -1, np.int32)
        gi[0, :j] = got
        ok, det = keep_set_ok(gi, np.array([j]), want_i, want_c, s[None], [n], [j])
        assert ok == expect, det
    small = 16                                 # J < 200: 99.5 % means identical
    s1 = np.linspace(10.0, -10.0, 64)
    s1[small] = s1[small - 1] - 1e-4
    w1_i, w1_c = oracle.select_keep(s1[None].astype(np.float32), [64], [small])
    gi = np.full((1, 64), -1, np.int32)
    gi[0, :small] = sorted(set(w1_i[0, :small]) - {small - 1} | {small})
    assert not keep_set_ok(gi, np.array([small]), w1_i, w1_c, s1[None], [64], [small])[0]
    s2 = np.linspace(10.0, -10.0, 64)          # clear gap: only the exact set passes
    w2_i, w2_c = oracle.select_keep(s2[None].astype(np.float32), [64], [small])
    gi = np.full((1, 64), -1, np.int32)
    gi[0, :small] = sorted(set(w2_i[0, :small]) - {small - 1} | {small})
    assert not keep_set_ok(gi, np.array([small]), w2_i, w2_c, s2[None], [64], [small])[0]
    assert not keep_set_ok(w2_i, np.array([small - 1]), w2_i, w2_c, s2[None], [64], [small])[0]
