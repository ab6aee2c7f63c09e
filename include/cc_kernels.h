/*
 * cc_kernels.h -- kernel-level entry points of the counter-causal refresh
 * library, each one step of the scoring pass on its own.  Same conventions
 * as cc.h (device pointers, caller-owned memory, asynchronous on `stream`,
 * host-side errors returned at once, device-side errors in the status word
 * read by cc_get_status).
 */
#ifndef CC_KERNELS_H_
#define CC_KERNELS_H_

#include "cc.h"

#ifdef __cplusplus
extern "C" {
#endif

/* y[rows][n] (fp32) = x[rows][k] (bf16) * w[n][k]^T (bf16, nn.Linear layout),
 * fp32 accumulation on the tensor cores.  n % 32 == 0, k % 8 == 0, 16-byte
 * aligned pointers.  This is the projection step of the layer the scoring
 * pass re-runs (Sec. 3.1). */
cc_status cc_linear_f32(const void *x, const void *w, float *y, int32_t rows, int32_t n,
                        int32_t k, void *stream);

/* Counter-causal attention (Sec. 3.1; Eq. 2 with the upper-triangular mask):
 * for every sequence b and slot i < seq_len[b] and query head t,
 *   out[b*cap+i][t] = softmax_{i<j<seq_len[b]}(q[b*cap+i][t] . k[b][j][t/G] / sqrt(dh)) v[b][j][t/G]
 * with G = n_q_heads / n_kv_heads, and out = 0 when no slot follows i.
 * q, out: bf16 [batch*cap][n_q_heads][head_dim]; k, v: bf16 [batch][cap][n_kv_heads][head_dim]
 * (post-RoPE keys as cached); seq_len: int32 [batch].  head_dim 64 or 128.
 * Rows i >= seq_len[b] of out are not written. */
cc_status cc_counter_causal_attention(const void *q, const void *k, const void *v,
                                      const int32_t *seq_len, void *out, int32_t batch,
                                      int32_t cap, int32_t n_q_heads, int32_t n_kv_heads,
                                      int32_t head_dim, void *stream);

/* The same counter-causal attention (Sec. 3.1, Eq. 2) with the queries and
 * the output carried as bf16 pairs hi + lo (hi = bf16(x), lo = bf16(x - hi),
 * x to about 2^-17 relative): q and out rows are
 * [hi: n_q_heads*head_dim | lo: n_q_heads*head_dim] bf16, so q and out are
 * [batch*cap][2*n_q_heads][head_dim].  On the tensor cores
 * S = q_hi k^T + q_lo k^T, and the probabilities enter P V as P_hi + P_lo.
 * This is the attention of the precise scoring pass (CC_SCORE_PRECISE).
 * k, v, seq_len and the shape rules are those of cc_counter_causal_attention;
 * rows i >= seq_len[b] of out are not written. */
cc_status cc_counter_causal_attention_split(const void *q, const void *k, const void *v,
                                            const int32_t *seq_len, void *out, int32_t batch,
                                            int32_t cap, int32_t n_q_heads, int32_t n_kv_heads,
                                            int32_t head_dim, void *stream);

#ifdef __cplusplus
}
#endif
#endif /* CC_KERNELS_H_ */
