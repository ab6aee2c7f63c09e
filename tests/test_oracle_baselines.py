"""Pins of the oracle's comparison scorers (Sec. 4: sliding window,
importance, H2O) by a library softmax, invariants and closed forms (no GPU)."""
import numpy as np
import pytest
import torch

import oracle
from tests._util import SMALL


def _keys(n, hkv, dh, seed):
    return np.random.default_rng(seed).normal(size=(n + 3, hkv, dh)) * 1.5


@pytest.mark.parametrize("n,hkv,q_lo", [(9, 2, 0), (12, 1, 5), (7, 3, 6)])
def test_colsums_match_torch_masked_softmax(n, hkv, q_lo):
    dh = 8
    k = _keys(n, hkv, dh, n * 10 + q_lo)
    got = oracle.key_attention_colsums(k, n, q_lo)
    want = np.zeros(n)
    kt = torch.from_numpy(k[:n])
    for g in range(hkv):
        logits = kt[:, g] @ kt[:, g].T / np.sqrt(dh)               # [query i, key j]
        mask = torch.arange(n)[None, :] <= torch.arange(n)[:, None]  # j <= i
        a = torch.softmax(logits.masked_fill(~mask, float("-inf")), dim=-1)
        want += a[q_lo:].sum(dim=0).numpy()
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-14)
    # every query row's weights sum to 1
    assert got.sum() == pytest.approx(hkv * (n - q_lo), rel=1e-12)
    # slots before q_lo are seen by every query; none gets weight from earlier rows
    assert np.all(got >= 0)


def test_equal_keys_give_harmonic_closed_forms():
    """All keys equal: query i spreads 1/(i+1) over slots 0..i, so
    c[j] = Hkv * sum_{i >= max(j, q_lo)} 1/(i+1); importance divides by
    Hkv * (n - j)."""
    n, hkv, dh, q_lo = 10, 2, 4, 3
    k = np.tile(np.array([0.3, -1.0, 0.5, 2.0]), (n, hkv, 1))
    c = oracle.key_attention_colsums(k, n, q_lo)
    for j in range(n):
        want = hkv * sum(1.0 / (i + 1) for i in range(max(j, q_lo), n))
        assert c[j] == pytest.approx(want, rel=1e-12)
    shape = SMALL.__class__(**{**SMALL.__dict__, "n_layers": 1, "n_kv_heads": hkv,
                               "n_q_heads": hkv, "head_dim": dh})
    cache = {"k": [k[None]], "seq_len": np.array([n])}
    imp = oracle.importance_scores(shape, cache)
    for j in range(n):
        want = sum(1.0 / (i + 1) for i in range(j, n)) / (n - j)
        assert imp[0, j] == pytest.approx(want, rel=1e-12)
    # the first slot, seen by every query, is the most important here
    assert np.argmax(imp[0, :n]) == 0


def test_recency_keeps_the_most_recent():
    pos = np.array([[3, 7, 8, 20, 21, 22, 0, 0]])
    cache = {"pos": pos, "seq_len": np.array([6])}
    s = oracle.recency_scores(cache)
    idx, cnt = oracle.select_keep(s.astype(np.float32), [6], [3])
    np.testing.assert_array_equal(idx[0, :cnt[0]], [3, 4, 5])
    assert np.all(s[0, 6:] == -np.inf)


def test_h2o_accumulates_over_layers_and_protects_recent():
    n, hkv, dh, recent = 11, 2, 8, 4
    shape = SMALL.__class__(**{**SMALL.__dict__, "n_layers": 3, "n_kv_heads": hkv,
                               "n_q_heads": 2 * hkv, "head_dim": dh})
    ks = [_keys(n, hkv, dh, 100 + l)[None] for l in range(3)]
    cache = {"k": ks, "seq_len": np.array([n])}
    acc = oracle.h2o_update(shape, cache, np.zeros((1, n + 3)), recent)
    want = sum(oracle.key_attention_colsums(ks[l][0], n, n - recent) for l in range(3))
    np.testing.assert_allclose(acc[0, :n], want, rtol=1e-12)
    assert acc[0, :n].sum() == pytest.approx(3 * hkv * recent, rel=1e-12)
    assert np.all(acc[0, n:] == 0)
    s = oracle.h2o_scores(acc, [n], recent)
    assert np.all(s[0, n - recent:n] == np.inf) and np.all(np.isfinite(s[0, :n - recent]))
    # running total: a second refresh adds the same amount again
    acc2 = oracle.h2o_update(shape, cache, acc.copy(), recent)
    np.testing.assert_allclose(acc2[0, :n], 2 * acc[0, :n], rtol=1e-12)
