// rowops.cu -- per-row kernels of the scoring pass: RMSNorm, embedding
// gather (full pass), the target-logit head and the log-sum-exp combine
// (Sec. 3.1: the score of row i is read off the logit of its own token x_i).
//
// One warp per cache row, rows = b*cap + i; rows with i >= seq_len[b] are
// skipped (the heads write -inf there).  All are HBM-bound streams with
// 16-byte vector accesses.
#include <algorithm>

#include "rowops.cuh"

namespace cc {

namespace {

constexpr int kWarps = 8;  // warps (rows) per block

CC_DEV bool row_valid(const int32_t *seq_len, int cap, int row, int &i, int &n) {
  const int b = row / cap;
  i = row - b * cap;
  n = seq_len[b];
  return i < n && n <= cap;
}

// Scoring a row range (cc_score_rows): only slots [rng_lo[b], rng_hi[b])
// are scored, every other slot gets -inf (so that the element-wise maximum of
// the ranks' buffers assembles the whole refresh); without a range (rng_hi
// null) every slot is scored.
CC_DEV bool in_score_range(const int32_t *rng_lo, const int32_t *rng_hi, int cap, int row) {
  if (!rng_hi) return true;
  const int b = row / cap, i = row - b * cap;
  return i >= rng_lo[b] && i < rng_hi[b];
}

// Row ranges of the inference cycle: slots [row_lo[b], seq_len[b]) (row_lo
// may be null: from slot 0).
CC_DEV bool row_in_range(const int32_t *seq_len, const int32_t *row_lo, int cap, int row) {
  int i, n;
  if (!row_valid(seq_len, cap, row, i, n)) return false;
  return !row_lo || i >= row_lo[row / cap];
}

// Warp w -> its cache row.  With a span (and row_lo), warps cover only the
// chunk rows: warp w takes slot row_lo[b] + k of sequence b = w / span,
// k = w % span; otherwise warp w takes row w of the whole cache.
CC_DEV bool warp_row(const int32_t *seq_len, const int32_t *row_lo, int cap, int rows, int span,
                     int w, int &row) {
  if (span > 0 && row_lo) {
    const int b = w / span;
    if (b >= rows / cap) return false;
    const int i = row_lo[b] + (w - b * span), n = seq_len[b];
    row = b * cap + i;
    return i >= 0 && i < n && n <= cap;
  }
  row = w;
  return row < rows && row_in_range(seq_len, row_lo, cap, row);
}

// 8 bf16 of a uint4 -> float
CC_DEV void unpack8(const uint4 &v, float *f) {
  f[0] = bf16_lo(v.x); f[1] = bf16_hi(v.x); f[2] = bf16_lo(v.y); f[3] = bf16_hi(v.y);
  f[4] = bf16_lo(v.z); f[5] = bf16_hi(v.z); f[6] = bf16_lo(v.w); f[7] = bf16_hi(v.w);
}

// Loads elements [e, e+8) of a row as float (bf16 or fp32 source).
template <bool IN_F32>
CC_DEV void load8(const void *row, int e, float *f) {
  if constexpr (IN_F32) {
    const float4 *p = reinterpret_cast<const float4 *>(reinterpret_cast<const float *>(row) + e);
    float4 a = p[0], b = p[1];
    f[0] = a.x; f[1] = a.y; f[2] = a.z; f[3] = a.w; f[4] = b.x; f[5] = b.y; f[6] = b.z; f[7] = b.w;
  } else {
    unpack8(*reinterpret_cast<const uint4 *>(reinterpret_cast<const __nv_bfloat16 *>(row) + e), f);
  }
}

// A lane's chunks of a row are e = lane * 8 + 256 * j; the loops below take
// them four at a time with every load issued before the arithmetic, so a warp
// keeps four (fp32: eight) 16-byte loads in flight instead of one (the sums
// run in the same order as one chunk at a time).
template <bool IN_F32>
CC_DEV float row_inv_rms(const void *row, int d, float eps, int lane) {
  float ss = 0.f;
  int e = lane * 8;
  for (; e + 3 * 256 < d; e += 4 * 256) {
    float f[4][8];
#pragma unroll
    for (int u = 0; u < 4; ++u) load8<IN_F32>(row, e + u * 256, f[u]);
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
      for (int k = 0; k < 8; ++k) ss = fmaf(f[u][k], f[u][k], ss);
  }
  for (; e < d; e += 256) {
    float f[8];
    load8<IN_F32>(row, e, f);
#pragma unroll
    for (int k = 0; k < 8; ++k) ss = fmaf(f[k], f[k], ss);
  }
  ss = warp_sum(ss);
  return rsqrtf(ss / (float)d + eps);
}

// Elements [e, e+8) of the normalised row: bf16(f * inv * gain) (fp16 with
// f16, a magnitude above kF16Max recorded in `over`), and with split the
// remainder at column offset d.
CC_DEV void store_norm8(__nv_bfloat16 *o, int d, int e, const float *f, const uint4 &g, float inv,
                        int split, bool f16, bool &over) {
  float gf[8], y[8];
  unpack8(g, gf);
#pragma unroll
  for (int k = 0; k < 8; ++k) y[k] = f[k] * inv * gf[k];
  uint4 v;
  v.x = pack_act2(y[0], y[1], f16, over);
  v.y = pack_act2(y[2], y[3], f16, over);
  v.z = pack_act2(y[4], y[5], f16, over);
  v.w = pack_act2(y[6], y[7], f16, over);
  *reinterpret_cast<uint4 *>(o + e) = v;
  if (split) {
    uint4 lo;
    lo.x = pack_bf16x2(y[0] - bf16_lo(v.x), y[1] - bf16_hi(v.x));
    lo.y = pack_bf16x2(y[2] - bf16_lo(v.y), y[3] - bf16_hi(v.y));
    lo.z = pack_bf16x2(y[4] - bf16_lo(v.z), y[5] - bf16_hi(v.z));
    lo.w = pack_bf16x2(y[6] - bf16_lo(v.w), y[7] - bf16_hi(v.w));
    *reinterpret_cast<uint4 *>(o + d + e) = lo;
  }
}

// out (bf16) = x * gain / rms(x).  split: the row holds [hi | lo] (2d values),
// hi = bf16(y), lo = bf16(y - hi), so hi + lo carries y to ~2^-17.  f16: out
// is fp16 instead (not with split); a value above kF16Max is reported.
template <bool IN_F32>
__global__ void __launch_bounds__(kWarps * 32)
    rmsnorm_kernel(const void *x, const __nv_bfloat16 *gain, __nv_bfloat16 *out, int d, float eps,
                   const int32_t *seq_len, const int32_t *row_lo, int cap, int rows, int span,
                   int split, int f16, unsigned *status) {
  const int lane = threadIdx.x & 31;
  int row;
  if (!warp_row(seq_len, row_lo, cap, rows, span, blockIdx.x * kWarps + (threadIdx.x >> 5), row))
    return;
  const size_t es = IN_F32 ? 4 : 2;
  const void *xr = reinterpret_cast<const uint8_t *>(x) + (size_t)row * d * es;
  const float inv = row_inv_rms<IN_F32>(xr, d, eps, lane);
  __nv_bfloat16 *o = out + (size_t)row * d * (split ? 2 : 1);
  bool over = false;
  int e = lane * 8;
  for (; e + 3 * 256 < d; e += 4 * 256) {
    float f[4][8];
    uint4 g[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      load8<IN_F32>(xr, e + u * 256, f[u]);
      g[u] = *reinterpret_cast<const uint4 *>(gain + e + u * 256);
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) store_norm8(o, d, e + u * 256, f[u], g[u], inv, split, f16, over);
  }
  for (; e < d; e += 256) {
    float f[8];
    load8<IN_F32>(xr, e, f);
    store_norm8(o, d, e, f, *reinterpret_cast<const uint4 *>(gain + e), inv, split, f16, over);
  }
  if (over) set_status(status, CC_ERR_RANGE);
}

// h (fp32) = embed[tokens[row]]
__global__ void __launch_bounds__(kWarps * 32)
    embed_kernel(const __nv_bfloat16 *embed, const int32_t *tokens, float *h, int d, int vocab,
                 const int32_t *seq_len, const int32_t *row_lo, int cap, int rows, int span,
                 unsigned *status) {
  const int lane = threadIdx.x & 31;
  int row;
  if (!warp_row(seq_len, row_lo, cap, rows, span, blockIdx.x * kWarps + (threadIdx.x >> 5), row))
    return;
  int tok = tokens[row];
  if (tok < 0 || tok >= vocab) {
    if (lane == 0) set_status(status, CC_ERR_DEVICE_ARG);
    tok = 0;
  }
  const __nv_bfloat16 *src = embed + (size_t)tok * d;
  float *dst = h + (size_t)row * d;
  for (int e = lane * 8; e < d; e += 256) {
    float f[8];
    unpack8(*reinterpret_cast<const uint4 *>(src + e), f);
    reinterpret_cast<float4 *>(dst + e)[0] = make_float4(f[0], f[1], f[2], f[3]);
    reinterpret_cast<float4 *>(dst + e)[1] = make_float4(f[4], f[5], f[6], f[7]);
  }
}

// out bf16 [row] = h fp32 [row] for the rows in range (H^(L-1) recorded by
// the inference cycle).
__global__ void __launch_bounds__(kWarps * 32)
    store_bf16_kernel(const float *h, __nv_bfloat16 *out, int d, const int32_t *seq_len,
                      const int32_t *row_lo, int cap, int rows, int span) {
  const int lane = threadIdx.x & 31;
  int row;
  if (!warp_row(seq_len, row_lo, cap, rows, span, blockIdx.x * kWarps + (threadIdx.x >> 5), row))
    return;
  const float *src = h + (size_t)row * d;
  __nv_bfloat16 *dst = out + (size_t)row * d;
  for (int e = lane * 8; e < d; e += 256) {
    float f[8];
    load8<true>(src, e, f);
    uint4 v;
    v.x = pack_bf16x2(f[0], f[1]);
    v.y = pack_bf16x2(f[2], f[3]);
    v.z = pack_bf16x2(f[4], f[5]);
    v.w = pack_bf16x2(f[6], f[7]);
    *reinterpret_cast<uint4 *>(dst + e) = v;
  }
}

// Inference cycle, start: sequence b (one block) appends count[b] slots after
// its seq_len[b] current ones: row_lo = seq_len, row_hi = seq_len + count;
// the chunk's tokens and positions (given, or continuing after the last
// cached position) are written into the cache.  A count outside
// [0, max_count] or past cap is reported and appends nothing.
__global__ void append_prepare_kernel(const int32_t *seq_len, const int32_t *count,
                                      const int32_t *tok_in, const int32_t *pos_in, int max_count,
                                      int32_t *tokens, int32_t *pos, int32_t *row_lo,
                                      int32_t *row_hi, int cap, unsigned *status) {
  const int b = blockIdx.x;
  const int lo = seq_len[b];
  int c = count ? count[b] : 1;   // no count array: one token each (a decode step)
  if (lo < 0 || lo > cap || c < 0 || c > max_count || lo + c > cap) {
    if (threadIdx.x == 0) set_status(status, CC_ERR_DEVICE_ARG);
    c = 0;   // nothing appended; seq_len is left as it was
  }
  if (threadIdx.x == 0) {
    row_lo[b] = lo;
    row_hi[b] = lo + c;
  }
  if (c == 0) return;
  const size_t base = (size_t)b * cap;
  const int next = lo > 0 ? pos[base + lo - 1] + 1 : 0;
  for (int i = threadIdx.x; i < c; i += blockDim.x) {
    tokens[base + lo + i] = tok_in[(size_t)b * max_count + i];
    pos[base + lo + i] = pos_in ? pos_in[(size_t)b * max_count + i] : next + i;
  }
}

__global__ void append_finish_kernel(int32_t *seq_len, const int32_t *row_hi, int batch) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b < batch) seq_len[b] = row_hi[b];
}

// Greedy decoding: the next token of sequence b is the first column of the
// largest logit over the column tiles' (max, column) pairs; -1 when the
// sequence appended nothing (row_hi == row_lo).
__global__ void argmax_combine_kernel(const float2 *part, int n_tiles, const int32_t *row_lo,
                                      const int32_t *row_hi, int batch, int32_t *next,
                                      float *best) {
  const int b = blockIdx.x;
  const int lane = threadIdx.x;
  float m = -INFINITY;
  int mi = 0x7FFFFFFF;
  if (row_hi[b] > row_lo[b]) {
    for (int t = lane; t < n_tiles; t += 32) {
      const float2 v = part[(size_t)b * n_tiles + t];
      const int idx = __float_as_int(v.y);
      if (idx >= 0 && (v.x > m || (v.x == m && idx < mi))) {
        m = v.x;
        mi = idx;
      }
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float om = __shfl_xor_sync(0xFFFFFFFFu, m, o);
    const int oi = __shfl_xor_sync(0xFFFFFFFFu, mi, o);
    if (om > m || (om == m && oi < mi)) {
      m = om;
      mi = oi;
    }
  }
  if (lane == 0) {
    next[b] = mi == 0x7FFFFFFF ? -1 : mi;
    if (best) best[b] = m;
  }
}

// score = -(RMSNorm(h) * g) . W_U[x_i] = -(sum h g W_U[x_i]) / rms(h), from
// the down projection's per-column-tile partials (sum h^2, sum h g W_U[x_i]);
// last valid slot +inf; past the end -inf.
__global__ void __launch_bounds__(kWarps * 32)
    head_logit_kernel(const float2 *part, int n_tiles, const int32_t *tokens, float *scores,
                      int d, int vocab, float eps, const int32_t *seq_len, int cap, int rows,
                      unsigned *status, const int32_t *rng_lo, const int32_t *rng_hi,
                      int keep_outside) {
  const int lane = threadIdx.x & 31;
  const int row = blockIdx.x * kWarps + (threadIdx.x >> 5);
  if (row >= rows) return;
  int i, n;
  // rows outside the range (another rank's) and past the sequence end: -inf,
  // or left as they are (keep_outside)
  if (!in_score_range(rng_lo, rng_hi, cap, row) || !row_valid(seq_len, cap, row, i, n)) {
    if (lane == 0 && !keep_outside) scores[row] = -INFINITY;
    return;
  }
  if (i == n - 1) {   // no future context: maximum surprise, always retained
    if (lane == 0) scores[row] = INFINITY;
    return;
  }
  const int tok = tokens[row];
  if ((tok < 0 || tok >= vocab) && lane == 0) set_status(status, CC_ERR_DEVICE_ARG);
  const float2 *pr = part + (size_t)row * n_tiles;
  float ss = 0.f, z = 0.f;
  for (int t = lane; t < n_tiles; t += 32) {
    const float2 v = pr[t];
    ss += v.x;
    z += v.y;
  }
  ss = warp_sum(ss);
  z = warp_sum(z);
  if (lane == 0) scores[row] = -(z * rsqrtf(ss / (float)d + eps));
}

// score = -(z_target - logsumexp) from per-tile (max, sum exp) partials.
__global__ void __launch_bounds__(kWarps * 32)
    lse_combine_kernel(const float2 *part, int n_tiles, const float *z_target, float *scores,
                       const int32_t *seq_len, int cap, int rows, const int32_t *rng_lo,
                       const int32_t *rng_hi, int keep_outside) {
  const int lane = threadIdx.x & 31;
  const int row = blockIdx.x * kWarps + (threadIdx.x >> 5);
  if (row >= rows) return;
  int i, n;
  // rows outside the range (another rank's) and past the sequence end: -inf,
  // or left as they are (keep_outside)
  if (!in_score_range(rng_lo, rng_hi, cap, row) || !row_valid(seq_len, cap, row, i, n)) {
    if (lane == 0 && !keep_outside) scores[row] = -INFINITY;
    return;
  }
  if (i == n - 1) {
    if (lane == 0) scores[row] = INFINITY;
    return;
  }
  const float2 *pr = part + (size_t)row * n_tiles;
  float m = -INFINITY;
  for (int t = lane; t < n_tiles; t += 32) m = fmaxf(m, pr[t].x);
  m = warp_max(m);
  float s = 0.f;
  for (int t = lane; t < n_tiles; t += 32) s += pr[t].y * __expf(pr[t].x - m);
  s = warp_sum(s);
  if (lane == 0) scores[row] = (m + __logf(s)) - z_target[row];
}

unsigned blocks_for(int rows) { return (unsigned)((rows + kWarps - 1) / kWarps); }

// warps of a row launch: one per cache row, or batch * span with a span
int warps_for(int rows, int cap, int span, const int32_t *row_lo) {
  return span > 0 && row_lo ? rows / cap * span : rows;
}

}  // namespace

cudaError_t launch_rmsnorm(const void *x, bool x_f32, const void *gain, void *out, int d, float eps,
                           const int32_t *seq_len, int cap, int rows, bool split, cudaStream_t st,
                           const int32_t *row_lo, int span, bool f16, unsigned *status) {
  if (rows <= 0) return cudaSuccess;
  if (split && f16) return cudaErrorInvalidValue;
  auto *g = reinterpret_cast<const __nv_bfloat16 *>(gain);
  auto *o = reinterpret_cast<__nv_bfloat16 *>(out);
  const unsigned blocks = blocks_for(warps_for(rows, cap, span, row_lo));
  if (x_f32)
    rmsnorm_kernel<true><<<blocks, kWarps * 32, 0, st>>>(x, g, o, d, eps, seq_len, row_lo, cap, rows,
                                                          span, split ? 1 : 0, f16 ? 1 : 0, status);
  else
    rmsnorm_kernel<false><<<blocks, kWarps * 32, 0, st>>>(x, g, o, d, eps, seq_len, row_lo, cap,
                                                           rows, span, split ? 1 : 0, f16 ? 1 : 0,
                                                           status);
  return cudaGetLastError();
}

cudaError_t launch_embed(const void *embed, const int32_t *tokens, float *h, int d, int vocab,
                         const int32_t *seq_len, int cap, int rows, unsigned *status,
                         cudaStream_t st, const int32_t *row_lo, int span) {
  if (rows <= 0) return cudaSuccess;
  embed_kernel<<<blocks_for(warps_for(rows, cap, span, row_lo)), kWarps * 32, 0, st>>>(
      reinterpret_cast<const __nv_bfloat16 *>(embed), tokens, h, d, vocab, seq_len, row_lo, cap,
      rows, span, status);
  return cudaGetLastError();
}

cudaError_t launch_store_bf16(const float *h, void *out, int d, const int32_t *seq_len,
                              const int32_t *row_lo, int cap, int rows, cudaStream_t st, int span) {
  if (rows <= 0) return cudaSuccess;
  store_bf16_kernel<<<blocks_for(warps_for(rows, cap, span, row_lo)), kWarps * 32, 0, st>>>(
      h, reinterpret_cast<__nv_bfloat16 *>(out), d, seq_len, row_lo, cap, rows, span);
  return cudaGetLastError();
}

cudaError_t launch_append_prepare(const int32_t *seq_len, const int32_t *count,
                                  const int32_t *tok_in, const int32_t *pos_in, int max_count,
                                  int32_t *tokens, int32_t *pos, int32_t *row_lo, int32_t *row_hi,
                                  int batch, int cap, unsigned *status, cudaStream_t st) {
  append_prepare_kernel<<<batch, 256, 0, st>>>(seq_len, count, tok_in, pos_in, max_count, tokens,
                                                pos, row_lo, row_hi, cap, status);
  return cudaGetLastError();
}

cudaError_t launch_argmax_combine(const float2 *part, int n_tiles, const int32_t *row_lo,
                                  const int32_t *row_hi, int batch, int32_t *next, float *best,
                                  cudaStream_t st) {
  argmax_combine_kernel<<<batch, 32, 0, st>>>(part, n_tiles, row_lo, row_hi, batch, next, best);
  return cudaGetLastError();
}

namespace {

// One layer's K/V as a slot-major copy for the tile attention: e4m3 codes ->
// bf16 or fp16 (exact: every e4m3 value is both), or bf16 -> fp16 (exact for
// magnitudes in [2^-14, 65504]; a larger one is reported), into rows
// b * cap + i, i < seq_end[b], from a slot-major, paged or head-major cache.
// One thread converts 16 elements of K and of V.  A paged row outside the
// pool is reported and skipped.
template <bool IN_FP8, bool OUT_F16>
__global__ void __launch_bounds__(256)
    kv_copy_kernel(const uint8_t *k, const uint8_t *v, KvLayout pg, int cap, int hkv, int dh,
                   const int32_t *seq_end, int batch, uint16_t *ko, uint16_t *vo,
                   unsigned *status) {
  const int chunks = hkv * dh / 16;   // 16-element chunks of one slot
  const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (long long)batch * cap * chunks) return;
  const long long row = idx / chunks;
  const int c = (int)(idx - row * chunks);
  const int b = (int)(row / cap), i = (int)(row - (long long)b * cap);
  if (i >= seq_end[b]) return;
  const int h = c * 16 / dh, e = c * 16 - h * dh;
  long long src;
  if (pg.head_major) {
    src = (((long long)b * hkv + h) * cap + i) * dh + e;
  } else {
    const long long r = kv_row(pg, cap, b, i);
    if (r < 0) {
      set_status(status, CC_ERR_DEVICE_ARG);
      return;
    }
    src = (r * hkv + h) * dh + e;
  }
  const size_t dst = (size_t)row * hkv * dh + (size_t)h * dh + e;
  bool over = false;
  auto convert = [&over](const uint8_t *in, uint16_t *out) {
    uint32_t o[8];
    if constexpr (IN_FP8) {
      const uint4 x = *reinterpret_cast<const uint4 *>(in);
      const uint32_t w[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
      for (int j = 0; j < 4; ++j)
#pragma unroll
        for (int hf = 0; hf < 2; ++hf) {   // two codes -> f16 pair (exact) [-> bf16 pair (exact)]
          uint32_t f2;
          asm("cvt.rn.f16x2.e4m3x2 %0, %1;" : "=r"(f2) : "h"((unsigned short)(w[j] >> (16 * hf))));
          if constexpr (OUT_F16) {
            o[j * 2 + hf] = f2;
          } else {
            const float2 f = __half22float2(*reinterpret_cast<const __half2 *>(&f2));
            o[j * 2 + hf] = pack_bf16x2(f.x, f.y);
          }
        }
    } else {   // bf16 -> fp16
      const uint4 *x = reinterpret_cast<const uint4 *>(in);
      const uint4 a = x[0], bq = x[1];
      const uint32_t w[8] = {a.x, a.y, a.z, a.w, bq.x, bq.y, bq.z, bq.w};
#pragma unroll
      for (int j = 0; j < 8; ++j) o[j] = pack_act2(bf16_lo(w[j]), bf16_hi(w[j]), true, over);
    }
    uint4 *d = reinterpret_cast<uint4 *>(out);
    d[0] = make_uint4(o[0], o[1], o[2], o[3]);
    d[1] = make_uint4(o[4], o[5], o[6], o[7]);
  };
  constexpr int EB = IN_FP8 ? 1 : 2;   // input bytes per element
  convert(k + src * EB, ko + dst);
  convert(v + src * EB, vo + dst);
  if (over) set_status(status, CC_ERR_RANGE);
}

// dst (fp16) = src (bf16), 8 values per thread and step (grid-stride).
__global__ void __launch_bounds__(256)
    bf16_to_f16_kernel(const uint4 *src, uint4 *dst, size_t n8, unsigned *status) {
  bool over = false;
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n8;
       i += (size_t)gridDim.x * blockDim.x) {
    const uint4 x = src[i];
    dst[i] = make_uint4(pack_act2(bf16_lo(x.x), bf16_hi(x.x), true, over),
                        pack_act2(bf16_lo(x.y), bf16_hi(x.y), true, over),
                        pack_act2(bf16_lo(x.z), bf16_hi(x.z), true, over),
                        pack_act2(bf16_lo(x.w), bf16_hi(x.w), true, over));
  }
  if (over) set_status(status, CC_ERR_RANGE);
}

}  // namespace

cudaError_t launch_kv_copy(const uint8_t *k, const uint8_t *v, bool in_fp8, bool out_f16,
                           const KvLayout &pg, int cap, int hkv, int dh, const int32_t *seq_end,
                           int batch, void *k_out, void *v_out, unsigned *status,
                           cudaStream_t st) {
  const long long n = (long long)batch * cap * (hkv * dh / 16);
  if (n <= 0) return cudaSuccess;
  if (!in_fp8 && !out_f16) return cudaErrorInvalidValue;   // bf16 -> bf16: no copy needed
  auto *ko = reinterpret_cast<uint16_t *>(k_out);
  auto *vo = reinterpret_cast<uint16_t *>(v_out);
  const unsigned blocks = (unsigned)((n + 255) / 256);
  if (in_fp8 && out_f16)
    kv_copy_kernel<true, true><<<blocks, 256, 0, st>>>(k, v, pg, cap, hkv, dh, seq_end, batch, ko,
                                                       vo, status);
  else if (in_fp8)
    kv_copy_kernel<true, false><<<blocks, 256, 0, st>>>(k, v, pg, cap, hkv, dh, seq_end, batch, ko,
                                                        vo, status);
  else
    kv_copy_kernel<false, true><<<blocks, 256, 0, st>>>(k, v, pg, cap, hkv, dh, seq_end, batch, ko,
                                                        vo, status);
  return cudaGetLastError();
}

cudaError_t launch_bf16_to_f16(const void *src, void *dst, size_t n, int sms, unsigned *status,
                               cudaStream_t st) {
  const size_t n8 = n / 8;
  if (n8 == 0) return cudaSuccess;
  const size_t want = (n8 + 255) / 256;
  const unsigned blocks = (unsigned)std::min<size_t>(want, (size_t)sms * 8);
  bf16_to_f16_kernel<<<blocks, 256, 0, st>>>(reinterpret_cast<const uint4 *>(src),
                                             reinterpret_cast<uint4 *>(dst), n8, status);
  return cudaGetLastError();
}

cudaError_t launch_append_finish(int32_t *seq_len, const int32_t *row_hi, int batch,
                                 cudaStream_t st) {
  append_finish_kernel<<<(batch + 255) / 256, 256, 0, st>>>(seq_len, row_hi, batch);
  return cudaGetLastError();
}

cudaError_t launch_head_logit(const float2 *part, int n_tiles, const int32_t *tokens,
                              float *scores, int d, int vocab, float eps, const int32_t *seq_len,
                              int cap, int rows, unsigned *status, cudaStream_t st,
                              const int32_t *rng_lo, const int32_t *rng_hi, bool keep_outside) {
  if (rows <= 0) return cudaSuccess;
  head_logit_kernel<<<blocks_for(rows), kWarps * 32, 0, st>>>(part, n_tiles, tokens, scores, d,
                                                             vocab, eps, seq_len, cap, rows,
                                                             status, rng_lo, rng_hi,
                                                             keep_outside ? 1 : 0);
  return cudaGetLastError();
}

cudaError_t launch_lse_combine(const float2 *part, int n_tiles, const float *z_target,
                               float *scores, const int32_t *seq_len, int cap, int rows,
                               cudaStream_t st, const int32_t *rng_lo, const int32_t *rng_hi,
                               bool keep_outside) {
  if (rows <= 0) return cudaSuccess;
  lse_combine_kernel<<<blocks_for(rows), kWarps * 32, 0, st>>>(part, n_tiles, z_target, scores,
                                                              seq_len, cap, rows, rng_lo, rng_hi,
                                                              keep_outside ? 1 : 0);
  return cudaGetLastError();
}

}  // namespace cc
