"""The restatements the fused GEMM epilogues compute, checked in fp64 against
the oracle's plain forms (no GPU).

* Logit head inside the last down projection: -(RMSNorm(x) * g) . W_U[t]
  = -(sum_j x_j g_j W_U[t, j]) * rsqrt(mean(x^2) + eps), the sums taken as
  per-column-tile partials and added in tile order.
* Post-attention RMSNorm across the O and gate/up epilogues:
  RMSNorm(h) W^T = rsqrt(mean(h^2) + eps) * ((h * g) W^T), with h * g rounded
  to bf16 for the GEMM instead of h * g / rms(h): the same relative rounding,
  so the same error against the exact product."""
import numpy as np

import oracle


def bf16(x):
    """Round fp64 values to the nearest bf16 (ties to even) via fp32 bits."""
    u = np.asarray(x, np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32).astype(np.float64)


def test_logit_head_from_tile_partials():
    r = np.random.default_rng(1)
    rows, d, vocab, tile = 37, 512, 300, 128
    x = r.normal(size=(rows, d)) * r.uniform(0.1, 10.0, size=(rows, 1))
    g = r.uniform(0.5, 1.5, size=d)
    w_u = r.normal(size=(vocab, d))
    tok = r.integers(0, vocab, size=rows)
    eps = 1e-5
    want = oracle.score_head(x, tok, g, w_u, "logit", eps)
    ss = np.zeros(rows)
    z = np.zeros(rows)
    for c0 in range(0, d, tile):   # per column tile, then in tile order
        xs = x[:, c0:c0 + tile]
        ss += np.sum(xs * xs, axis=1)
        z += np.sum(xs * g[c0:c0 + tile] * w_u[tok, c0:c0 + tile], axis=1)
    got = -(z / np.sqrt(ss / d + eps))
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-12)


def test_norm_scale_moves_past_the_gemm():
    r = np.random.default_rng(2)
    rows, d, n = 64, 256, 96
    h = r.normal(size=(rows, d)) * r.uniform(0.01, 50.0, size=(rows, 1))
    g = r.uniform(0.5, 1.5, size=d)
    w = bf16(r.normal(size=(n, d)) * 0.05)
    eps = 1e-5
    exact = oracle.rms_norm(h, g, eps) @ w.T
    rs = 1.0 / np.sqrt(np.mean(h * h, axis=1, keepdims=True) + eps)
    np.testing.assert_allclose(rs * ((h * g) @ w.T), exact, rtol=1e-12, atol=1e-12)
    # rounding the GEMM input: normalised-then-rounded vs rounded-then-scaled
    err_plain = np.abs(bf16(oracle.rms_norm(h, g, eps)) @ w.T - exact)
    err_fused = np.abs(rs * (bf16(h * g) @ w.T) - exact)
    scale = np.sqrt(np.mean(exact * exact))
    e1, e2 = np.mean(err_plain) / scale, np.mean(err_fused) / scale
    assert 0.0 < e1 < 1e-2 and 0.0 < e2 < 1e-2
    assert 0.8 < e2 / e1 < 1.25   # the same rounding error, row scale aside
