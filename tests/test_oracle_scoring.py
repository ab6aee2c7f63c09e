"""Pins of the oracle's counter-causal scoring (Sec. 3.1) by closed-form
special cases and invariants (no GPU)."""
import copy

import numpy as np
import pytest

import oracle
from tests._util import SMALL, causal_cache, small_model

SEQ = [13, 9, 1]
CAP = 16


@pytest.fixture(scope="module")
def model():
    return small_model(SMALL, seed=5)


@pytest.fixture(scope="module")
def cache(model):
    return causal_cache(SMALL, model, SEQ, CAP, seed=5)


def _last(w):
    return w["layers"][SMALL.n_layers - 1]


def _rms(x):
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + SMALL.rms_eps)


def test_last_slot_is_max_surprise(model, cache):
    s = oracle.score_layer(SMALL, model, cache)
    for b, n in enumerate(SEQ):
        assert s[b, n - 1] == np.inf
        assert np.all(np.isfinite(s[b, :n - 1]))
        assert np.all(s[b, n:] == -np.inf)


def test_closed_form_no_attention_no_mlp(model, cache):
    """Wo = 0 and W_down = 0: the layer is the identity, so the score is
    -RMSNorm(H_i) . W_U[x_i] (the row's own token)."""
    w = copy.deepcopy(model)
    w["layers"][-1]["wo"][:] = 0
    w["layers"][-1]["w_down"][:] = 0
    s = oracle.score_layer(SMALL, w, cache)
    for b, n in enumerate(SEQ):
        h = cache["h_last"][b, :n].astype(np.float64)
        want = -np.sum(_rms(h) * w["lm_head"][cache["tokens"][b, :n]], axis=-1)
        np.testing.assert_allclose(s[b, :n - 1], want[:n - 1], rtol=1e-12)


def test_closed_form_uniform_attention(model, cache):
    """Wq = 0 gives uniform weights over the strictly later slots; with
    W_down = 0 the layer output is H_i + concat_t(mean_{j>i} V_j[t // G]) Wo^T."""
    w = copy.deepcopy(model)
    w["layers"][-1]["wq"][:] = 0
    w["layers"][-1]["w_down"][:] = 0
    s = oracle.score_layer(SMALL, w, cache)
    g = SMALL.n_q_heads // SMALL.n_kv_heads
    v = cache["v"][-1]
    for b, n in enumerate(SEQ):
        for i in range(n - 1):
            o = np.concatenate([v[b, i + 1:n, t // g].astype(np.float64).mean(axis=0)
                                for t in range(SMALL.n_q_heads)])
            h = cache["h_last"][b, i] + w["layers"][-1]["wo"].astype(np.float64) @ o
            want = -np.sum(_rms(h) * w["lm_head"][cache["tokens"][b, i]])
            assert s[b, i] == pytest.approx(want, rel=1e-11)


def test_no_leakage_from_past_or_self_kv(model, cache):
    """Score i depends on K/V only at slots j > i: changing K/V at slots <= i
    and H at other slots leaves it bit-identical; changing K at j > i does not."""
    b, n, i = 0, SEQ[0], 6
    base = oracle.score_layer(SMALL, model, cache)[b, i]
    c2 = copy.deepcopy(cache)
    r = np.random.default_rng(0)
    c2["k"][-1][b, :i + 1] += r.normal(size=c2["k"][-1][b, :i + 1].shape).astype(np.float32)
    c2["v"][-1][b, :i + 1] += r.normal(size=c2["v"][-1][b, :i + 1].shape).astype(np.float32)
    c2["h_last"][b, i + 1:n] += 1.0
    c2["tokens"][b, i + 1:n] = (c2["tokens"][b, i + 1:n] + 1) % SMALL.vocab
    assert oracle.score_layer(SMALL, model, c2)[b, i] == base
    c3 = copy.deepcopy(cache)
    c3["k"][-1][b, i + 1] += 1.0
    assert oracle.score_layer(SMALL, model, c3)[b, i] != base


def test_prefix_drop_invariance(model, cache):
    """Dropping slots < i0 (original positions kept) leaves later scores unchanged."""
    b, n, i0 = 0, SEQ[0], 5
    full = oracle.score_layer(SMALL, model, cache)[b, i0:n]
    c2 = {"k": [x[b:b + 1, i0:] for x in cache["k"]], "v": [x[b:b + 1, i0:] for x in cache["v"]],
          "tokens": cache["tokens"][b:b + 1, i0:], "pos": cache["pos"][b:b + 1, i0:],
          "h_last": cache["h_last"][b:b + 1, i0:], "seq_len": np.array([n - i0])}
    np.testing.assert_allclose(oracle.score_layer(SMALL, model, c2)[0, :n - i0], full,
                               rtol=1e-13)


def test_batch_equals_single_sequences(model, cache):
    both = oracle.score_layer(SMALL, model, cache, mode="logprob")
    for b in range(len(SEQ)):
        one = {k: ([x[b:b + 1] for x in v] if isinstance(v, list) else v[b:b + 1])
               for k, v in cache.items()}
        np.testing.assert_array_equal(oracle.score_layer(SMALL, model, one, mode="logprob")[0],
                                      both[b])


def test_row_subset_equals_all_rows(model, cache):
    allr = oracle.score_full(SMALL, model, cache)
    rows = [[0, 4, 12], [8], []]
    sub = oracle.score_full(SMALL, model, cache, rows=rows)
    for b, r in enumerate(rows):
        np.testing.assert_array_equal(sub[b, r], allr[b, r])


def _permute_heads(w, cache, perm_q_within, perm_kv):
    """Relabel heads: KV groups by perm_kv, query heads inside a group by
    perm_q_within, with the matching Wq row blocks and Wo column blocks."""
    hq, hkv, dh = SMALL.n_q_heads, SMALL.n_kv_heads, SMALL.head_dim
    g = hq // hkv
    w2, c2 = copy.deepcopy(w), copy.deepcopy(cache)
    new_of_old_q = []
    for t_new in range(hq):
        grp_new, pos_new = divmod(t_new, g)
        new_of_old_q.append(perm_kv[grp_new] * g + perm_q_within[pos_new])
    for lw in w2["layers"]:
        wq = lw["wq"].reshape(hq, dh, -1)
        lw["wq"] = wq[new_of_old_q].reshape(hq * dh, -1)
        wo = lw["wo"].reshape(-1, hq, dh)
        lw["wo"] = wo[:, new_of_old_q].reshape(-1, hq * dh)
    c2["k"] = [x[:, :, perm_kv] for x in cache["k"]]
    c2["v"] = [x[:, :, perm_kv] for x in cache["v"]]
    return w2, c2


def test_gqa_head_permutation_invariance(model, cache):
    base = oracle.score_layer(SMALL, model, cache)
    w2, c2 = _permute_heads(model, cache, perm_q_within=[1, 0], perm_kv=[1, 0])
    got = oracle.score_layer(SMALL, w2, c2)
    fin = np.isfinite(base)
    np.testing.assert_array_equal(np.isfinite(got), fin)
    np.testing.assert_allclose(got[fin], base[fin], rtol=1e-11)
    # a mismatched relabelling (K/V heads swapped, queries not) does change scores
    c3 = copy.deepcopy(cache)
    c3["k"] = [x[:, :, [1, 0]] for x in cache["k"]]
    assert not np.allclose(oracle.score_layer(SMALL, model, c3)[fin], base[fin])


def test_full_pass_with_one_layer_equals_fast_mode():
    """With L = 1 the last layer's input is the embedding, so the full pass and
    the fast single-layer approximation coincide (Sec. 3.1)."""
    shape1 = SMALL.__class__(**{**SMALL.__dict__, "n_layers": 1})
    w = small_model(shape1, seed=8)
    c = causal_cache(shape1, w, [11, 4], 12, seed=8)
    np.testing.assert_allclose(oracle.score_full(shape1, w, c), oracle.score_layer(shape1, w, c),
                               rtol=1e-12)
    # with L = 2 they differ
    w2 = small_model(SMALL, seed=8)
    c2 = causal_cache(SMALL, w2, [11], 12, seed=8)
    a, b = oracle.score_full(SMALL, w2, c2), oracle.score_layer(SMALL, w2, c2)
    assert not np.allclose(a[0, :10], b[0, :10])


def test_rope_shift_invariance(model):
    """Shifting every original position by D (cache rebuilt by the causal
    forward at the shifted positions) leaves the scores unchanged: RoPE only
    sees relative offsets."""
    n = 10
    toks = np.random.default_rng(3).integers(0, SMALL.vocab, size=n)

    def built(offset):
        pos = np.arange(n) + offset
        fw = oracle.causal_forward(SMALL, model, toks, pos)
        return {"k": [x[None] for x in fw["k"]], "v": [x[None] for x in fw["v"]],
                "h_last": fw["h_last"][None], "tokens": toks[None], "pos": pos[None],
                "seq_len": np.array([n])}
    s0 = oracle.score_full(SMALL, model, built(0))
    s1 = oracle.score_full(SMALL, model, built(100003))
    np.testing.assert_allclose(s1[0, :n - 1], s0[0, :n - 1], rtol=1e-9)
    s2 = oracle.score_layer(SMALL, model, built(7))
    np.testing.assert_allclose(s2[0, :n - 1], oracle.score_layer(SMALL, model, built(0))[0, :n - 1],
                               rtol=1e-9)


def test_worked_example_by_hand():
    """A three-slot cache small enough to score with a pencil (Sec. 3.1, the
    surprise of each cached token given only its future; Algorithm
    DoMemRefresh, keep the J highest and compact).  One layer, d = 2, one
    head, eps = 0.  W_q = 0 makes every attention score 0, so slot i averages
    the values of slots i+1 .. n-1; W_o = I adds that average to h_i; W_down = 0
    silences the MLP; gains are 1; W_U rows are e_0, e_1 and e_0 + e_1.

      slot  token  h_i       v_i        o_i            h_i + o_i   RMSNorm
      0     0      (1, 1)    (5, 5)     (v1+v2)/2=(0,2)   (1, 3)     (1, 3)/sqrt(5)
      1     1      (1, -1)   (1, 1)     v2 = (-1, 3)      (0, 2)     (0, sqrt(2))
      2     2      (2, 0)    (-1, 3)    no future: +inf
      3     (stale slot past n = 3: -inf, never read)

    logit scores: -W_U[x_i] . RMSNorm = -1/sqrt(5), -sqrt(2), +inf.
    log-prob scores: logsumexp(z_i) - z_i[x_i] with z_0 = (1, 3, 4)/sqrt(5),
    z_1 = (0, sqrt(2), sqrt(2)).  Budget J = 2 keeps slots 0 and 2 in both
    modes; compaction moves slot 2 to slot 1."""
    import math
    from synth.configs import ModelShape
    shape = ModelShape(n_layers=1, d_model=2, n_q_heads=1, n_kv_heads=1, head_dim=2, d_ff=2,
                       vocab=3, rope_theta=1e4, rms_eps=0.0)
    eye, zero, ones = np.eye(2), np.zeros((2, 2)), np.ones(2)
    h = np.array([[1.0, 1.0], [1.0, -1.0], [2.0, 0.0], [7.0, 7.0]])
    lw = {"attn_norm": ones, "wq": zero, "wk": eye, "wv": eye, "wo": eye, "mlp_norm": ones,
          "w_gate": eye, "w_up": eye, "w_down": zero}
    w = {"layers": [lw], "final_norm": ones, "lm_head": np.array([[1.0, 0], [0, 1.0], [1.0, 1.0]]),
         "embed": np.array([[1.0, 1.0], [1.0, -1.0], [2.0, 0.0]])}
    v = np.array([[5.0, 5.0], [1.0, 1.0], [-1.0, 3.0], [100.0, -100.0]])[None, :, None, :]
    k = np.arange(8.0).reshape(1, 4, 1, 2)
    cache = {"k": [k], "v": [v], "tokens": np.array([[0, 1, 2, 0]]),
             "pos": np.array([[0, 1, 2, 3]]), "seq_len": np.array([3]), "h_last": h[None]}

    def lse(*z):
        return math.log(sum(math.exp(t) for t in z))

    s5, s2 = math.sqrt(5.0), math.sqrt(2.0)
    want = {"logit": [-1 / s5, -s2],
            "logprob": [lse(1 / s5, 3 / s5, 4 / s5) - 1 / s5, lse(0.0, s2, s2) - s2]}
    for mode, (w0, w1) in want.items():
        for got in (oracle.score_layer(shape, w, cache, mode),
                    oracle.score_full(shape, w, cache, mode)):   # embed rows = h: same pass
            np.testing.assert_allclose(got[0, :2], [w0, w1], rtol=1e-14, atol=1e-14)
            assert got[0, 2] == np.inf and got[0, 3] == -np.inf
            idx, cnt = oracle.select_keep(got.astype(np.float32), [3], [2])
            assert cnt.tolist() == [2] and idx[0, :2].tolist() == [0, 2]
    np.testing.assert_array_equal(oracle.compact(cache["tokens"], idx, cnt)[0, :2], [0, 2])
    np.testing.assert_array_equal(oracle.compact(v, idx, cnt)[0, :2, 0], v[0, [0, 2], 0])
    np.testing.assert_array_equal(oracle.compact(h[None], idx, cnt)[0, :2], h[[0, 2]])


def test_logprob_scores_are_a_distribution_over_the_target_token(model, cache):
    """In the fast pass a slot's hidden state comes from H^(L-1) and its own
    K/V are never attended (only later slots are), so its token id enters the
    score only as the target: re-scoring one slot with every vocabulary entry
    as its token must give probabilities exp(-score) that sum to 1 (the
    surprise is -log P(x_i | its future), Sec. 3.1), and logit-mode scores
    differ from them by one constant per slot."""
    b, n = 0, SEQ[0]
    for i in (0, 4, n - 2):
        lp, lg = [], []
        for v in range(SMALL.vocab):
            c = copy.deepcopy(cache)
            c["tokens"][b, i] = v
            lp.append(oracle.score_layer(SMALL, model, c, "logprob", rows=[[i], None, None])[b, i])
            lg.append(oracle.score_layer(SMALL, model, c, "logit", rows=[[i], None, None])[b, i])
        lp, lg = np.array(lp), np.array(lg)
        assert abs(np.exp(-lp).sum() - 1.0) < 1e-12
        np.testing.assert_allclose(lp - lg, np.full(SMALL.vocab, (lp - lg)[0]), rtol=0, atol=1e-12)
