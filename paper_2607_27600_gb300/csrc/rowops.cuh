// rowops.cuh -- per-row kernels of the scoring pass.
#pragma once
#include "cc_common.cuh"

namespace cc {

// out bf16 [rows][d] = x * gain / sqrt(mean(x^2) + eps); x bf16 or fp32 [rows][d].
// split: out rows are [hi | lo] bf16 [rows][2d] with hi + lo ~= the fp32 value.
// Row kernels visit rows b*cap + i with row_lo[b] <= i < seq_len[b] (row_lo
// null: from 0).  span > 0 (with row_lo): seq_len[b] - row_lo[b] <= span, and
// the launch has batch * span warps instead of one per cache row.
// f16: out is fp16 [rows][d] instead (not with split); a value above 65504 in
// magnitude sets CC_ERR_RANGE in status.
cudaError_t launch_rmsnorm(const void *x, bool x_f32, const void *gain, void *out, int d, float eps,
                           const int32_t *seq_len, int cap, int rows, bool split, cudaStream_t st,
                           const int32_t *row_lo = nullptr, int span = 0, bool f16 = false,
                           unsigned *status = nullptr);
// h fp32 [rows][d] = embed[tokens[row]]
cudaError_t launch_embed(const void *embed, const int32_t *tokens, float *h, int d, int vocab,
                         const int32_t *seq_len, int cap, int rows, unsigned *status,
                         cudaStream_t st, const int32_t *row_lo = nullptr, int span = 0);
// out bf16 [rows][d] = h fp32 (H^(L-1) recorded by the inference cycle)
cudaError_t launch_store_bf16(const float *h, void *out, int d, const int32_t *seq_len,
                              const int32_t *row_lo, int cap, int rows, cudaStream_t st,
                              int span = 0);
// Inference cycle: row_lo = seq_len, row_hi = seq_len + count; the chunk's
// tokens and positions written into the cache slots [row_lo, row_hi).
cudaError_t launch_append_prepare(const int32_t *seq_len, const int32_t *count,
                                  const int32_t *tok_in, const int32_t *pos_in, int max_count,
                                  int32_t *tokens, int32_t *pos, int32_t *row_lo, int32_t *row_hi,
                                  int batch, int cap, unsigned *status, cudaStream_t st);
// seq_len = row_hi
// One layer of the cache copied for the tile attention, slot-major
// [batch * cap][hkv][dh] for the slots i < seq_end[b] (dh a multiple of 16):
// e4m3 codes (in_fp8) as bf16 or fp16 (out_f16) values, exact either way, or
// bf16 as fp16 (exact for magnitudes in [2^-14, 65504]; a larger one sets
// CC_ERR_RANGE).  bf16 to bf16 is refused (cudaErrorInvalidValue).
cudaError_t launch_kv_copy(const uint8_t *k, const uint8_t *v, bool in_fp8, bool out_f16,
                           const KvLayout &pg, int cap, int hkv, int dh, const int32_t *seq_end,
                           int batch, void *k_out, void *v_out, unsigned *status,
                           cudaStream_t st);
// dst (fp16) = src (bf16) for n elements (n a multiple of 8, both 16-byte
// aligned); a finite value above 65504 in magnitude sets CC_ERR_RANGE.
cudaError_t launch_bf16_to_f16(const void *src, void *dst, size_t n, int sms, unsigned *status,
                               cudaStream_t st);
cudaError_t launch_append_finish(int32_t *seq_len, const int32_t *row_hi, int batch,
                                 cudaStream_t st);
// next[b] = first column of the largest logit over the (max, column) tile
// pairs part[b][n_tiles] (-1 when sequence b appended nothing); best[b] = it
cudaError_t launch_argmax_combine(const float2 *part, int n_tiles, const int32_t *row_lo,
                                  const int32_t *row_hi, int batch, int32_t *next, float *best,
                                  cudaStream_t st);
// scores[row] = -(final-norm(h) . lm_head[tokens[row]]) from the per-tile
// partials part[row][n_tiles] = (sum h^2, sum h * gain * lm_head[tokens[row]])
// of the fused down projection; +inf at the last slot.  rng_lo / rng_hi
// (device [batch], or null): only slots [rng_lo[b], rng_hi[b]) are scored,
// the others get -inf (keep_outside: keep their values).
cudaError_t launch_head_logit(const float2 *part, int n_tiles, const int32_t *tokens,
                              float *scores, int d, int vocab, float eps, const int32_t *seq_len,
                              int cap, int rows, unsigned *status, cudaStream_t st,
                              const int32_t *rng_lo = nullptr, const int32_t *rng_hi = nullptr,
                              bool keep_outside = false);
// scores[row] = logsumexp - z_target, +inf at the last slot (ranges as above)
cudaError_t launch_lse_combine(const float2 *part, int n_tiles, const float *z_target,
                               float *scores, const int32_t *seq_len, int cap, int rows,
                               cudaStream_t st, const int32_t *rng_lo = nullptr,
                               const int32_t *rng_hi = nullptr, bool keep_outside = false);

}  // namespace cc
