"""Pins of the oracle's building blocks against library routines, closed
forms and brute force (no GPU)."""
import math

import numpy as np
import pytest
import scipy.special
import torch
import torch.nn.functional as F

import oracle


def rng(seed=0):
    return np.random.default_rng(seed)


def test_rms_norm_matches_torch():
    x = rng(1).normal(size=(5, 33)) * 3.0
    g = rng(2).normal(size=33)
    want = F.rms_norm(torch.from_numpy(x), (33,), weight=torch.from_numpy(g), eps=1e-5).numpy()
    np.testing.assert_allclose(oracle.rms_norm(x, g, 1e-5), want, rtol=1e-12, atol=1e-12)


def test_rms_norm_closed_form():
    # [3, 4]: mean square 12.5 -> divide by sqrt(12.5)
    np.testing.assert_allclose(oracle.rms_norm(np.array([3.0, 4.0]), np.ones(2), 0.0),
                               [3 / math.sqrt(12.5), 4 / math.sqrt(12.5)], rtol=1e-15)


def test_rope_is_complex_rotation():
    """Rotate-half RoPE == multiplying z_k = x_k + i x_{k+dh/2} by exp(i pos w_k)."""
    dh, theta = 16, 1e4
    x = rng(3).normal(size=(7, 3, dh))
    pos = np.array([0, 1, 5, 77, 1000, 4095, 131071])
    w = 1.0 / theta ** (np.arange(0, dh, 2) / dh)
    z = x[..., : dh // 2] + 1j * x[..., dh // 2:]
    zr = z * np.exp(1j * pos[:, None, None] * w[None, None, :])
    want = np.concatenate([zr.real, zr.imag], axis=-1)
    np.testing.assert_allclose(oracle.rope(x, pos, theta), want, rtol=1e-10, atol=1e-10)


def test_rope_relative_position():
    """<rope(q, p), rope(k, p')> depends only on p - p'."""
    dh = 32
    q, k = rng(4).normal(size=(1, 1, dh)), rng(5).normal(size=(1, 1, dh))
    def dot(p1, p2):
        return float(np.sum(oracle.rope(q, np.array([p1]), 5e5) * oracle.rope(k, np.array([p2]), 5e5)))
    assert dot(10, 3) == pytest.approx(dot(1010, 1003), rel=1e-9, abs=1e-9)
    assert dot(0, 0) == pytest.approx(float(np.sum(q * k)), rel=1e-12)
    assert abs(dot(10, 3) - dot(10, 4)) > 1e-6


def _sdpa_counter_causal(q, k, v, rows, n):
    """torch SDPA with an explicit boolean mask (key j allowed iff rows[r] < j < n)."""
    hq, hkv = q.shape[1], k.shape[1]
    kk = torch.from_numpy(k[:n]).repeat_interleave(hq // hkv, dim=1).permute(1, 0, 2)
    vv = torch.from_numpy(v[:n]).repeat_interleave(hq // hkv, dim=1).permute(1, 0, 2)
    qq = torch.from_numpy(q).permute(1, 0, 2)
    j = torch.arange(n)
    mask = (j[None, :] > torch.from_numpy(np.asarray(rows))[:, None])
    out = F.scaled_dot_product_attention(qq, kk, vv, attn_mask=mask)
    return out.permute(1, 0, 2).numpy()


@pytest.mark.parametrize("hq,hkv,dh", [(4, 2, 16), (7, 1, 8), (3, 3, 4), (8, 2, 64)])
def test_counter_causal_attention_matches_sdpa(hq, hkv, dh):
    n, cap = 23, 30
    r = rng(hq * 100 + dh)
    q = r.normal(size=(n, hq, dh))
    k, v = r.normal(size=(cap, hkv, dh)) * 2, r.normal(size=(cap, hkv, dh))
    rows = np.arange(n - 1)                        # the last row has no key: SDPA gives NaN
    got = oracle.counter_causal_attention(q[rows], k, v, rows, n)
    np.testing.assert_allclose(got, _sdpa_counter_causal(q[rows], k, v, rows, n),
                               rtol=1e-10, atol=1e-12)


def test_counter_causal_attention_brute_force():
    """Scalar loops on a 5-token, 2-dim, single-head case."""
    r = rng(9)
    n, dh = 5, 2
    q, k, v = r.normal(size=(n, 1, dh)), r.normal(size=(n, 1, dh)), r.normal(size=(n, 1, dh))
    got = oracle.counter_causal_attention(q, k, v, np.arange(n), n)
    for i in range(n):
        w = [math.exp(sum(q[i, 0, c] * k[j, 0, c] for c in range(dh)) / math.sqrt(dh))
             for j in range(i + 1, n)]
        for c in range(dh):
            want = (sum(wj * v[j, 0, c] for wj, j in zip(w, range(i + 1, n))) / sum(w)) if w else 0.0
            assert got[i, 0, c] == pytest.approx(want, rel=1e-12, abs=1e-14)


def test_counter_causal_attention_closed_forms():
    r = rng(11)
    n, hq, hkv, dh = 9, 4, 2, 8
    q = r.normal(size=(n, hq, dh)) * 5
    k, v = r.normal(size=(n, hkv, dh)), r.normal(size=(n, hkv, dh))
    out = oracle.counter_causal_attention(q, k, v, np.arange(n), n)
    # row n-2 sees only key n-1 -> exactly V[n-1] of its KV head
    for t in range(hq):
        np.testing.assert_array_equal(out[n - 2, t], v[n - 1, t // 2])
    # last row: empty key set -> 0
    np.testing.assert_array_equal(out[n - 1], 0.0)
    # K == 0 -> uniform weights -> mean of the later values
    out0 = oracle.counter_causal_attention(q, np.zeros_like(k), v, np.arange(n), n)
    for i in range(n - 1):
        for t in range(hq):
            np.testing.assert_allclose(out0[i, t], v[i + 1:n, t // 2].mean(axis=0), rtol=1e-12)


def test_counter_causal_attention_ignores_stale_slots():
    """Slots >= n (stale, even non-finite) never reach the output."""
    r = rng(12)
    n, cap = 6, 10
    q = r.normal(size=(n, 2, 4))
    k, v = r.normal(size=(cap, 1, 4)), r.normal(size=(cap, 1, 4))
    k2, v2 = k.copy(), v.copy()
    k2[n:], v2[n:] = np.nan, np.inf
    a = oracle.counter_causal_attention(q, k, v, np.arange(n), n)
    b = oracle.counter_causal_attention(q, k2, v2, np.arange(n), n)
    np.testing.assert_array_equal(a, b)


def test_causal_attention_matches_sdpa():
    r = rng(13)
    n, hq, hkv, dh = 17, 6, 2, 8
    q, k, v = r.normal(size=(n, hq, dh)), r.normal(size=(n, hkv, dh)), r.normal(size=(n, hkv, dh))
    kk = torch.from_numpy(k).repeat_interleave(3, dim=1).permute(1, 0, 2)
    vv = torch.from_numpy(v).repeat_interleave(3, dim=1).permute(1, 0, 2)
    want = F.scaled_dot_product_attention(torch.from_numpy(q).permute(1, 0, 2), kk, vv,
                                          is_causal=True).permute(1, 0, 2).numpy()
    np.testing.assert_allclose(oracle.causal_attention(q, k, v), want, rtol=1e-10, atol=1e-12)


def test_swiglu_scalar_case():
    # m = 2, Wg = 1.5, Wu = 0.5, Wd = 3: gate 3, silu(3) = 3 / (1 + e^-3), up 1
    lw = {"w_gate": np.array([[1.5]]), "w_up": np.array([[0.5]]), "w_down": np.array([[3.0]])}
    silu3 = 3.0 * 0.9525741268224334           # logistic(3) = 0.95257412682243...
    np.testing.assert_allclose(oracle.swiglu_mlp(np.array([[2.0]]), lw), [[silu3 * 1.0 * 3.0]],
                               rtol=1e-14)


def test_swiglu_matches_torch_silu():
    r = rng(14)
    m = r.normal(size=(3, 6))
    lw = {"w_gate": r.normal(size=(5, 6)), "w_up": r.normal(size=(5, 6)),
          "w_down": r.normal(size=(6, 5))}
    t = {k: torch.from_numpy(v) for k, v in lw.items()}
    mt = torch.from_numpy(m)
    want = (F.silu(mt @ t["w_gate"].T) * (mt @ t["w_up"].T)) @ t["w_down"].T
    np.testing.assert_allclose(oracle.swiglu_mlp(m, lw), want.numpy(), rtol=1e-12)


def test_score_head_closed_form():
    # h = [3, 4] -> u = h / sqrt(12.5); W_U[x] = [1, -1] -> z = -1/sqrt(12.5); score = -z
    h = np.array([[3.0, 4.0]])
    lm = np.array([[0.0, 0.0], [1.0, -1.0]])
    s = oracle.score_head(h, np.array([1]), np.ones(2), lm, "logit", 0.0)
    assert s[0] == pytest.approx(1 / math.sqrt(12.5), rel=1e-15)


def test_score_head_logprob_matches_scipy():
    r = rng(15)
    h = r.normal(size=(4, 10))
    lm = r.normal(size=(37, 10))
    tok = np.array([0, 5, 36, 5])
    got = oracle.score_head(h, tok, np.ones(10), lm, "logprob", 1e-6, vocab_chunk=8)
    u = oracle.rms_norm(h, np.ones(10), 1e-6)
    lsm = scipy.special.log_softmax(u @ lm.T, axis=-1)
    np.testing.assert_allclose(got, -lsm[np.arange(4), tok], rtol=1e-12)
    # logit-mode and log-prob-mode scores differ by exactly the log-normaliser
    lg = oracle.score_head(h, tok, np.ones(10), lm, "logit", 1e-6)
    np.testing.assert_allclose(got - lg, scipy.special.logsumexp(u @ lm.T, axis=-1), rtol=1e-12)


def test_sensitivity_bf16_rounding_matches_torch():
    from tests.study_fullpass_precision import bf16
    r = rng(21)
    x = np.concatenate([r.normal(size=1000) * 10.0 ** r.integers(-6, 6, size=1000),
                        [1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, -(1.0 + 2.0 ** -8), 0.0, -0.0]])
    want = torch.from_numpy(x.astype(np.float32)).to(torch.bfloat16).double().numpy()
    np.testing.assert_array_equal(bf16(x), want)


# Llama-3.1 scaling parameters (factor, low_freq_factor, high_freq_factor,
# original_max_position) at Llama-3's theta and head_dim
LLAMA31_SCALING = (8.0, 1.0, 4.0, 8192)


def test_rope_scaling_none_is_plain_rope():
    inv = oracle.rope_inv_freq(128, 5e5)
    np.testing.assert_array_equal(inv, 5e5 ** (-np.arange(64) / 64.0))
    np.testing.assert_array_equal(oracle.rope_angles(np.array([3]), 128, 5e5),
                                  oracle.rope_angles(np.array([3]), 128, 5e5, None))


def test_rope_scaling_bands():
    """Three bands by wavelength w = 2 pi / inv_freq: below orig/high the
    frequency is unchanged, above orig/low it is divided by the factor, and in
    between the ratio scaled/plain is an affine function of inv_freq that
    reaches 1 at the short edge and 1/factor at the long edge (continuity)."""
    factor, low, high, orig = LLAMA31_SCALING
    plain = oracle.rope_inv_freq(128, 5e5)
    scaled = oracle.rope_inv_freq(128, 5e5, LLAMA31_SCALING)
    w = 2 * np.pi / plain
    short, long_ = w < orig / high, w > orig / low
    mid = ~short & ~long_
    assert short.sum() > 10 and long_.sum() > 10 and mid.sum() >= 3
    np.testing.assert_array_equal(scaled[short], plain[short])
    np.testing.assert_allclose(scaled[long_], plain[long_] / factor, rtol=1e-15)
    r = scaled[mid] / plain[mid]
    assert np.all((r > 1 / factor) & (r < 1))
    slope, icpt = np.polyfit(plain[mid], r, 1)
    np.testing.assert_allclose(slope * plain[mid] + icpt, r, rtol=1e-12)
    edge_short = 2 * np.pi / (orig / high)     # inv_freq at w = orig / high
    edge_long = 2 * np.pi / (orig / low)
    assert slope * edge_short + icpt == pytest.approx(1.0, rel=1e-12)
    assert slope * edge_long + icpt == pytest.approx(1 / factor, rel=1e-12)
    # monotone: frequencies still decrease with k
    assert np.all(np.diff(scaled) < 0)


def test_projection_bias_closed_form():
    """Wq = 0 with a q bias b: every row's queries are RoPE(b) at its own
    position, so attention weights are softmax(RoPE(b_t, pos_i) . K_j / sqrt(dh))
    over j > i; with W_down = 0 the layer output follows in closed form."""
    from tests._util import SMALL, small_model, causal_cache
    shape = SMALL.__class__(**{**SMALL.__dict__, "qkv_bias": True, "n_layers": 1})
    w = small_model(shape, seed=31)
    c = causal_cache(shape, w, [9], 10, seed=31)
    lw = w["layers"][0]
    assert "bq" in lw and np.abs(lw["bq"]).max() > 0.1
    lw["wq"][:] = 0
    lw["w_down"][:] = 0
    s = oracle.score_layer(shape, w, c)
    g = shape.n_q_heads // shape.n_kv_heads
    dh, half = shape.head_dim, shape.head_dim // 2
    k, v = c["k"][0][0].astype(np.float64), c["v"][0][0].astype(np.float64)
    for i in range(8):
        o = []
        for t in range(shape.n_q_heads):
            b = lw["bq"][t * dh:(t + 1) * dh].astype(np.float64)
            z = (b[:half] + 1j * b[half:]) * np.exp(1j * i * shape.rope_theta ** (-np.arange(half) / half))
            q = np.concatenate([z.real, z.imag])
            logits = np.array([q @ k[j, t // g] for j in range(i + 1, 9)]) / np.sqrt(dh)
            p = np.exp(logits - logits.max())
            o.append((p / p.sum()) @ v[i + 1:9, t // g])
        h = c["h_last"][0, i] + lw["wo"].astype(np.float64) @ np.concatenate(o)
        u = h / np.sqrt(np.mean(h * h) + shape.rms_eps)
        assert s[0, i] == pytest.approx(-u @ w["lm_head"][c["tokens"][0, i]], rel=1e-10)


def test_biased_scaled_model_is_rope_shift_invariant():
    """q/k biases added before RoPE, scaled frequencies: the scores still see
    only relative offsets (a bias added after the rotation would not)."""
    from tests._util import SMALL, small_model
    shape = SMALL.__class__(**{**SMALL.__dict__, "qkv_bias": True,
                               "rope_scaling": (4.0, 1.0, 4.0, 32)})
    w = small_model(shape, seed=32)
    n = 10
    toks = np.random.default_rng(4).integers(0, shape.vocab, size=n)

    def built(offset):
        pos = np.arange(n) + offset
        fw = oracle.causal_forward(shape, w, toks, pos)
        return {"k": [x[None] for x in fw["k"]], "v": [x[None] for x in fw["v"]],
                "h_last": fw["h_last"][None], "tokens": toks[None], "pos": pos[None],
                "seq_len": np.array([n])}
    s0 = oracle.score_full(shape, w, built(0))
    np.testing.assert_allclose(oracle.score_full(shape, w, built(5003))[0, :n - 1],
                               s0[0, :n - 1], rtol=1e-9)
    # the scaling and the biases do change the scores
    plain = SMALL.__class__(**{**shape.__dict__, "rope_scaling": None})
    assert not np.allclose(oracle.score_full(plain, w, built(0))[0, :n - 1], s0[0, :n - 1])
    w0 = {**w, "layers": [{k_: v_ for k_, v_ in lw.items() if not k_.startswith("b")}
                          for lw in w["layers"]]}
    assert not np.allclose(oracle.score_full(shape, w0, built(0))[0, :n - 1], s0[0, :n - 1])
