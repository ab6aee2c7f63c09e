"""Pins of the oracle's inference cycle in pre-fill (Algorithm
CacheManagedInference / DoInference, chunked mode): memory-augmented causal
attention (Eq. 3) and the chunk append (no GPU)."""
import copy
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
from tests._util import SMALL, small_model


def _empty_cache(shape, cap, batch=1):
    return {"k": [np.zeros((batch, cap, shape.n_kv_heads, shape.head_dim)) for _ in range(shape.n_layers)],
            "v": [np.zeros((batch, cap, shape.n_kv_heads, shape.head_dim)) for _ in range(shape.n_layers)],
            "tokens": np.zeros((batch, cap), np.int32), "pos": np.zeros((batch, cap), np.int32),
            "seq_len": np.zeros(batch, np.int32), "h_last": np.zeros((batch, cap, shape.d_model))}


@pytest.mark.parametrize("hq,hkv,n0,h", [(4, 2, 7, 5), (3, 1, 0, 6), (2, 2, 11, 1)])
def test_memory_causal_attention_matches_sdpa(hq, hkv, n0, h):
    r = np.random.default_rng(hq * 10 + n0)
    dh = 8
    q = r.normal(size=(h, hq, dh))
    k, v = r.normal(size=(n0 + h + 3, hkv, dh)), r.normal(size=(n0 + h + 3, hkv, dh))
    got = oracle.memory_causal_attention(q, k, v, n0)
    kk = torch.from_numpy(k[:n0 + h]).repeat_interleave(hq // hkv, dim=1).permute(1, 0, 2)
    vv = torch.from_numpy(v[:n0 + h]).repeat_interleave(hq // hkv, dim=1).permute(1, 0, 2)
    j = torch.arange(n0 + h)
    mask = j[None, :] <= (n0 + torch.arange(h))[:, None]     # memory all visible, chunk causal
    want = F.scaled_dot_product_attention(torch.from_numpy(q).permute(1, 0, 2), kk, vv,
                                          attn_mask=mask).permute(1, 0, 2).numpy()
    np.testing.assert_allclose(got, want, rtol=1e-10, atol=1e-12)
    if n0 == 0:
        np.testing.assert_array_equal(got, oracle.causal_attention(q, k[:h], v[:h]))


def _model(shape, seed):
    return small_model(shape, seed=seed)


def test_append_into_empty_cache_is_the_causal_forward():
    w = _model(SMALL, 41)
    toks = np.random.default_rng(41).integers(0, SMALL.vocab, size=9)
    c = _empty_cache(SMALL, 12)
    x = oracle.append_chunk(SMALL, w, c, 0, toks)
    fw = oracle.causal_forward(SMALL, w, toks, np.arange(9))
    for l in range(SMALL.n_layers):
        np.testing.assert_allclose(c["k"][l][0, :9], fw["k"][l], rtol=1e-12, atol=1e-14)
        np.testing.assert_allclose(c["v"][l][0, :9], fw["v"][l], rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(c["h_last"][0, :9], fw["h_last"], rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(x, fw["h_final"], rtol=1e-12, atol=1e-14)
    assert c["seq_len"][0] == 9
    np.testing.assert_array_equal(c["tokens"][0, :9], toks)
    np.testing.assert_array_equal(c["pos"][0, :9], np.arange(9))


def test_chunk_by_chunk_equals_one_append():
    """Without a refresh between them, appending 5 + 1 + 7 tokens leaves the
    same cache as appending all 13 at once (and as the causal forward)."""
    w = _model(SMALL, 42)
    toks = np.random.default_rng(42).integers(0, SMALL.vocab, size=13)
    c1, c2 = _empty_cache(SMALL, 16), _empty_cache(SMALL, 16)
    for a, e in ((0, 5), (5, 6), (6, 13)):
        x1 = oracle.append_chunk(SMALL, w, c1, 0, toks[a:e])
    x2 = oracle.append_chunk(SMALL, w, c2, 0, toks)
    for l in range(SMALL.n_layers):
        np.testing.assert_allclose(c1["k"][l], c2["k"][l], rtol=1e-11, atol=1e-13)
        np.testing.assert_allclose(c1["v"][l], c2["v"][l], rtol=1e-11, atol=1e-13)
    np.testing.assert_allclose(c1["h_last"], c2["h_last"], rtol=1e-11, atol=1e-13)
    np.testing.assert_allclose(x1, x2[6:], rtol=1e-11, atol=1e-13)
    np.testing.assert_array_equal(c1["pos"], c2["pos"])


def test_append_after_compaction_brute_force():
    """One layer, memory compacted to 5 of 9 slots (original positions kept),
    then a 3-token chunk: each chunk row's output by scalar loops over the
    kept memory slots and the chunk slots up to its own; positions continue
    after the last kept position; stale slots past the memory are unseen."""
    shape = SMALL.__class__(**{**SMALL.__dict__, "n_layers": 1})
    w = _model(shape, 43)
    r = np.random.default_rng(43)
    c = _empty_cache(shape, 16)
    oracle.append_chunk(shape, w, c, 0, r.integers(0, shape.vocab, size=9))
    keep = np.array([[1, 2, 4, 6, 8] + [-1] * 11])
    cnt = np.array([5])
    for key in ("tokens", "pos", "h_last"):
        c[key] = oracle.compact(c[key], keep, cnt)
    c["k"][0] = oracle.compact(c["k"][0], keep, cnt)
    c["v"][0] = oracle.compact(c["v"][0], keep, cnt)
    c["seq_len"] = cnt.copy()
    c["k"][0][0, 5:] = np.nan          # stale slots: overwritten or never read
    c["v"][0][0, 8:] = np.inf
    mem_k, mem_v = c["k"][0][0, :5].copy(), c["v"][0][0, :5].copy()
    chunk = r.integers(0, shape.vocab, size=3)
    x = oracle.append_chunk(shape, w, c, 0, chunk)
    np.testing.assert_array_equal(c["pos"][0, :8], [1, 2, 4, 6, 8, 9, 10, 11])
    lw = w["layers"][0]
    dh, half, g = shape.head_dim, shape.head_dim // 2, shape.n_q_heads // shape.n_kv_heads
    rows = [w["embed"][t].astype(np.float64) for t in chunk]

    def rot(vec, p):
        z = (vec[:half] + 1j * vec[half:]) * np.exp(1j * p * shape.rope_theta ** (-np.arange(half) / half))
        return np.concatenate([z.real, z.imag])

    def norm(vec, gain):
        return vec / math.sqrt(sum(t * t for t in vec) / len(vec) + shape.rms_eps) * gain
    ks, vs = [], []
    for ri, e in enumerate(rows):
        a = norm(e, lw["attn_norm"])
        kr = (lw["wk"] @ a).reshape(shape.n_kv_heads, dh)
        ks.append(np.stack([rot(kr[t], 9 + ri) for t in range(shape.n_kv_heads)]))
        vs.append((lw["wv"] @ a).reshape(shape.n_kv_heads, dh))
    for ri, e in enumerate(rows):
        a = norm(e, lw["attn_norm"])
        qr = (lw["wq"] @ a).reshape(shape.n_q_heads, dh)
        o = []
        for t in range(shape.n_q_heads):
            qt = rot(qr[t], 9 + ri)
            keys = [mem_k[j, t // g] for j in range(5)] + [ks[j][t // g] for j in range(ri + 1)]
            vals = [mem_v[j, t // g] for j in range(5)] + [vs[j][t // g] for j in range(ri + 1)]
            logit = [float(qt @ kk) / math.sqrt(dh) for kk in keys]
            mx = max(logit)
            p = [math.exp(s - mx) for s in logit]
            o.append(sum(pi * vv for pi, vv in zip(p, vals)) / sum(p))
        hh = e + lw["wo"] @ np.concatenate(o)
        m = norm(hh, lw["mlp_norm"])
        gt, up = lw["w_gate"] @ m, lw["w_up"] @ m
        want = hh + lw["w_down"] @ (gt / (1 + np.exp(-gt)) * up)
        np.testing.assert_allclose(x[ri], want, rtol=1e-10, atol=1e-12)
    assert np.all(np.isfinite(c["k"][0][0, :8])) and c["seq_len"][0] == 8


def test_decode_steps_equal_the_causal_forward():
    """Greedy decoding step by step (append one token, LM head, argmax) gives,
    at every step, the argmax of the causal forward's final hidden state at
    the last position of the whole sequence so far; an argmax pin against
    the logits themselves."""
    shape = SMALL
    w = _model(shape, 44)
    prompt = list(np.random.default_rng(44).integers(0, shape.vocab, size=6))
    c = _empty_cache(shape, 16)
    oracle.append_chunk(shape, w, c, 0, prompt[:-1])
    seq = list(prompt)
    tok = prompt[-1]
    for _ in range(4):
        nxt, best, logits = oracle.decode_step(shape, w, c, [tok])
        fw = oracle.causal_forward(shape, w, np.array(seq), np.arange(len(seq)))
        u = fw["h_final"][-1] / np.sqrt(np.mean(fw["h_final"][-1] ** 2) + shape.rms_eps)
        z = (u * w["final_norm"]) @ w["lm_head"].astype(np.float64).T
        np.testing.assert_allclose(logits[0], z, rtol=1e-10, atol=1e-12)
        assert nxt[0] == int(np.argmax(z)) and best[0] == pytest.approx(z.max(), rel=1e-12)
        assert c["seq_len"][0] == len(seq)
        tok = int(nxt[0])
        seq.append(tok)
