// gemm.cu -- persistent tcgen05 GEMM  D[rows, N] = A[rows, K] * B[N, K]^T
// (bf16 operands, fp32 accumulation in TMEM) with the epilogues the
// counter-causal layer needs (Sec. 3.1, the "standard" layer re-run over the
// cache): RoPE'd query projection, residual adds, SwiGLU, LM-head
// log-sum-exp partials, and the last residual add fused with the logit head.
//
// Rows are the cache slots of a ragged batch: sequence b owns rows
// b*cap + [0, seq_len[b]).  Only row tiles that hold valid slots are visited
// (seq_len is read on the device).
//
// CTA = 6 warps, one CTA per SM, persistent over (row tile, column tile):
//   warp 0      TMA producer (A 128x64 and B 256x64 bf16 tiles, 128B swizzle)
//   warp 1      TMEM owner + single-thread tcgen05.mma issuer (M=128, N=256, K=16)
//   warps 2..5  epilogue: tcgen05.ld of the accumulator (one row per thread)
// Two 256-column accumulators in TMEM let the epilogue of one tile overlap
// the main loop of the next.
// Large launches run as CTA pairs (clusters of two, cta_group::2): one
// M = 256, N = 256 product per pair, each CTA staging its own 128 A rows and
// half of the B tile, so a CTA moves 32 KB instead of 48 KB through L2 and
// shared memory per 128 x 256 x 64 block of its output.
#include "gemm.cuh"

#include <algorithm>

namespace cc {

namespace {

// BN: the widest column tile (256); a launch uses TBN = 256 or, for narrow
// problems (less than one wave of 256-column tiles), 128.
constexpr int BM = 128, BN = 256, BK = 64, ST = 4;
// CTA pairs (one 256 x 256 product per pair, each CTA holding 128 A rows and
// 128 B rows of a k-block): 16 + 16 KB ring slots, six of them, which the
// kernel fills and drains two per barrier stage
constexpr int ST_PAIR = 6;
constexpr int A_BYTES = BM * BK * 2;   // 16 KB
constexpr int B_BYTES = BN * BK * 2;   // 32 KB: shared-memory stage of the widest B tile
constexpr int kThreads = 192;
constexpr int kMaxBatch = 1024;
// fp32 epilogues stage each 32 x 32 accumulator chunk of a warp in shared
// memory (rows padded to 36 floats: 16-byte aligned, conflict-free float4
// accesses in both directions)
constexpr int kStageLd = 36;
constexpr int kStageBytes = 4 * 32 * kStageLd * 4;   // the four epilogue warps
constexpr size_t kPrefixBytes = ((kMaxBatch + 1) * sizeof(int) + 15) & ~size_t(15);
__host__ __device__ constexpr size_t stages(bool pair) { return pair ? ST_PAIR : ST; }
__host__ __device__ constexpr size_t b_stage_bytes(bool pair) { return pair ? B_BYTES / 2 : B_BYTES; }
__host__ __device__ constexpr size_t ring_bytes(bool pair) { return stages(pair) * (A_BYTES + b_stage_bytes(pair)); }
__host__ __device__ constexpr size_t smem_bytes(bool pair) {
  return 1024 /*align slack*/ + ring_bytes(pair) + 256 + kPrefixBytes + kStageBytes;
}
static_assert(smem_bytes(false) <= 232448 && smem_bytes(true) <= 232448, "shared memory");

// RoPE'd bf16 store of one accumulator tile row: destination columns
// [col0, col0 + TBN) of out (row stride ldo, n_dest columns in all), each tile
// holding TBN / head_dim whole heads; rotate-half pairs (k, k + dh/2); the
// bias (optional) is added before the rotation.
// F8: the destination is an e4m3 cache (one byte per element, the value
// times qscale = 1 / the layer's scale; pack_e4m3x2).
// orow: the output row (grow, or the cache row of a paged K destination; < 0: skip)
// Address of output column c of row `orow` (element size EB), or with a
// head-major cache destination (hm) of head c / head_dim's vector of slot
// grow % cap (32-column chunks never straddle two heads).
template <int EB>
CC_DEV uint8_t *out_at(const GemmParams &p, uint8_t *base, long long orow, int ldo, bool hm,
                       int grow, int c) {
  if (hm) {
    const int b = grow / p.cap, i = grow - b * p.cap;
    return base + ((((size_t)b * p.pg.hkv + c / p.head_dim) * p.cap + i) * p.head_dim +
                   c % p.head_dim) * EB;
  }
  return base + ((size_t)orow * ldo + c) * EB;
}

// The RMSNorm scale 1 / rms(x) of A row `grow` when the A rows are
// unnormalised (x * gain, with the per-column-tile partial sums of x^2 in
// row_ss, summed in a fixed order), else 1.
CC_DEV float row_rms_scale(const GemmParams &p, int grow, bool valid) {
  if (!p.row_ss || !valid) return 1.f;
  const float *pr = p.row_ss + (size_t)grow * p.n_ss;
  float ss = 0.f;
  for (int t = 0; t < p.n_ss; ++t) ss += pr[t];
  return rsqrtf(ss / (float)p.ss_d + p.eps);
}

// lo_off > 0 (bf16 only): also the lo half of each value, bf16(y - hi), at
// element offset lo_off of the row (the precise pass's [hi | lo] queries).
// rs: scale of the accumulator (before the bias and the rotation).  With
// p.out_f16 (not F8, lo_off 0) the values are written as fp16.
template <int TBN, bool F8 = false>
CC_DEV void rope_store(const GemmParams &p, uint32_t tacc, int grow, long long orow, bool valid,
                       void *out_base, int ldo, const __nv_bfloat16 *bias, int col0, int n_dest,
                       float qscale = 1.f, bool hm = false, int lo_off = 0, float rs = 1.f) {
  const int half = p.head_dim >> 1;
  valid = valid && orow >= 0;
  const uint32_t pos = valid ? (uint32_t)p.pos[grow] : 0u;
  uint8_t *base = reinterpret_cast<uint8_t *>(out_base);
#pragma unroll 1
  for (int hb = 0; hb < TBN; hb += p.head_dim) {
#pragma unroll 1
    for (int c0 = 0; c0 < half; c0 += 32) {
      uint32_t x1[32], x2[32];
      tmem_ld32(tacc + hb + c0, x1);
      tmem_ld32(tacc + hb + half + c0, x2);
      tmem_ld_wait();
      int col = col0 + hb + c0;
      if (!valid || col >= n_dest) continue;
      uint32_t bb1[16], bb2[16];   // bias pairs of columns col.. and col+half.. (0 if none)
#pragma unroll
      for (int v = 0; v < 4; ++v) {
        uint4 u1 = make_uint4(0, 0, 0, 0), u2 = make_uint4(0, 0, 0, 0);
        if (bias) {
          u1 = reinterpret_cast<const uint4 *>(bias + col)[v];
          u2 = reinterpret_cast<const uint4 *>(bias + col + half)[v];
        }
        bb1[v * 4] = u1.x; bb1[v * 4 + 1] = u1.y; bb1[v * 4 + 2] = u1.z; bb1[v * 4 + 3] = u1.w;
        bb2[v * 4] = u2.x; bb2[v * 4 + 1] = u2.y; bb2[v * 4 + 2] = u2.z; bb2[v * 4 + 3] = u2.w;
      }
      uint32_t o1[16], o2[16];
      [[maybe_unused]] uint32_t l1[16], l2[16];
      [[maybe_unused]] bool over = false;
#pragma unroll
      for (int k = 0; k < 32; k += 2) {
        float c_a, s_a, c_b, s_b;
        rope_cs(pos, p.turns[c0 + k], c_a, s_a);
        rope_cs(pos, p.turns[c0 + k + 1], c_b, s_b);
        float a1 = fmaf(__uint_as_float(x1[k]), rs, bf16_lo(bb1[k / 2]));
        float a2 = fmaf(__uint_as_float(x2[k]), rs, bf16_lo(bb2[k / 2]));
        float b1 = fmaf(__uint_as_float(x1[k + 1]), rs, bf16_hi(bb1[k / 2]));
        float b2 = fmaf(__uint_as_float(x2[k + 1]), rs, bf16_hi(bb2[k / 2]));
        if constexpr (F8) {   // two codes per pair, four per word
          const uint32_t e1 = pack_e4m3x2((a1 * c_a - a2 * s_a) * qscale,
                                          (b1 * c_b - b2 * s_b) * qscale);
          const uint32_t e2 = pack_e4m3x2((a2 * c_a + a1 * s_a) * qscale,
                                          (b2 * c_b + b1 * s_b) * qscale);
          if ((k & 2) == 0) {
            o1[k / 4] = e1;
            o2[k / 4] = e2;
          } else {
            o1[k / 4] |= e1 << 16;
            o2[k / 4] |= e2 << 16;
          }
        } else {
          const float y1a = a1 * c_a - a2 * s_a, y1b = b1 * c_b - b2 * s_b;
          const float y2a = a2 * c_a + a1 * s_a, y2b = b2 * c_b + b1 * s_b;
          o1[k / 2] = pack_act2(y1a, y1b, p.out_f16, over);
          o2[k / 2] = pack_act2(y2a, y2b, p.out_f16, over);
          l1[k / 2] = pack_bf16x2(y1a - bf16_lo(o1[k / 2]), y1b - bf16_hi(o1[k / 2]));
          l2[k / 2] = pack_bf16x2(y2a - bf16_lo(o2[k / 2]), y2b - bf16_hi(o2[k / 2]));
        }
      }
      if constexpr (!F8)
        if (over) set_status(p.status, CC_ERR_RANGE);
      constexpr int EB = F8 ? 1 : 2;
      uint4 *d1 = reinterpret_cast<uint4 *>(out_at<EB>(p, base, orow, ldo, hm, grow, col));
      uint4 *d2 = reinterpret_cast<uint4 *>(out_at<EB>(p, base, orow, ldo, hm, grow, col + half));
#pragma unroll
      for (int v = 0; v < 2 * EB; ++v) {   // 32 elements: 64 bytes bf16, 32 e4m3
        d1[v] = make_uint4(o1[v * 4], o1[v * 4 + 1], o1[v * 4 + 2], o1[v * 4 + 3]);
        d2[v] = make_uint4(o2[v * 4], o2[v * 4 + 1], o2[v * 4 + 2], o2[v * 4 + 3]);
      }
      if constexpr (!F8) {
        if (lo_off > 0) {
          uint4 *e1 = reinterpret_cast<uint4 *>(out_at<EB>(p, base, orow, ldo, hm, grow, col + lo_off));
          uint4 *e2 = reinterpret_cast<uint4 *>(
              out_at<EB>(p, base, orow, ldo, hm, grow, col + half + lo_off));
#pragma unroll
          for (int v = 0; v < 4; ++v) {
            e1[v] = make_uint4(l1[v * 4], l1[v * 4 + 1], l1[v * 4 + 2], l1[v * 4 + 3]);
            e2[v] = make_uint4(l2[v * 4], l2[v * 4 + 1], l2[v * 4 + 2], l2[v * 4 + 3]);
          }
        }
      }
    }
  }
}

// Plain bf16 store (+ optional bias) of one accumulator tile row; F8: e4m3
// codes of (value + bias) * qscale instead.
template <int TBN, bool F8 = false>
CC_DEV void plain_store(const GemmParams &p, uint32_t tacc, int grow, long long orow, bool valid,
                        void *out_base, int ldo, const __nv_bfloat16 *bias, int col0, int n_dest,
                        float qscale = 1.f, bool hm = false) {
  constexpr int EB = F8 ? 1 : 2;
  valid = valid && orow >= 0;
  uint8_t *base = reinterpret_cast<uint8_t *>(out_base);
#pragma unroll 1
  for (int c = 0; c < TBN / 32; ++c) {
    uint32_t r[32];
    tmem_ld32(tacc + c * 32, r);
    tmem_ld_wait();
    const int col = col0 + c * 32;
    if (!valid || col >= n_dest) continue;
    uint32_t bb[16];
#pragma unroll
    for (int v = 0; v < 4; ++v) {
      const uint4 u = bias ? reinterpret_cast<const uint4 *>(bias + col)[v] : make_uint4(0, 0, 0, 0);
      bb[v * 4] = u.x; bb[v * 4 + 1] = u.y; bb[v * 4 + 2] = u.z; bb[v * 4 + 3] = u.w;
    }
    uint32_t o[16];
#pragma unroll
    for (int k = 0; k < 32; k += 2) {
      const float y0 = __uint_as_float(r[k]) + bf16_lo(bb[k / 2]);
      const float y1 = __uint_as_float(r[k + 1]) + bf16_hi(bb[k / 2]);
      if constexpr (F8) {
        const uint32_t e = pack_e4m3x2(y0 * qscale, y1 * qscale);
        if ((k & 2) == 0) o[k / 4] = e;
        else o[k / 4] |= e << 16;
      } else {
        o[k / 2] = pack_bf16x2(y0, y1);
      }
    }
    uint4 *d = reinterpret_cast<uint4 *>(out_at<EB>(p, base, orow, ldo, hm, grow, col));
#pragma unroll
    for (int v = 0; v < 2 * EB; ++v)   // 32 elements: 64 bytes bf16, 32 e4m3
      d[v] = make_uint4(o[v * 4], o[v * 4 + 1], o[v * 4 + 2], o[v * 4 + 3]);
  }
}

// Cache row of workspace row grow = b * cap + i (paged: through the block
// table); a bad page is reported and the row skipped (-1).
CC_DEV long long cache_row(const GemmParams &p, int grow, bool valid) {
  const int b = grow / p.cap;
  const long long r = kv_row(p.pg, p.cap, b, grow - b * p.cap);
  if (r < 0 && valid) set_status(p.status, CC_ERR_DEVICE_ARG);
  return r;
}

// Chunk c of a warp's accumulator (32 rows x 32 columns, one row per lane as
// tcgen05.ld delivers it) into the warp's staging tile; afterwards lane l
// reads row 4 * i + l / 8 (i = 0..7), columns 4 * (l % 8) .. +4, so global
// reads and writes run along rows (whole 128-byte lines per 8 lanes).
CC_DEV void stage_chunk(float *stage, const uint32_t (&r)[32], int lane) {
  float4 *srow = reinterpret_cast<float4 *>(stage + lane * kStageLd);
#pragma unroll
  for (int v = 0; v < 8; ++v)
    srow[v] = make_float4(__uint_as_float(r[v * 4]), __uint_as_float(r[v * 4 + 1]),
                          __uint_as_float(r[v * 4 + 2]), __uint_as_float(r[v * 4 + 3]));
  __syncwarp();
}

// Sum over the 8 lanes that share a row in the staged layout.
CC_DEV float row8_sum(float v) {
  v += __shfl_xor_sync(0xFFFFFFFFu, v, 1);
  v += __shfl_xor_sync(0xFFFFFFFFu, v, 2);
  v += __shfl_xor_sync(0xFFFFFFFFu, v, 4);
  return v;
}

// The final residual row x = out + acc of one tile (never stored): partial
// sum of x^2 and partial dot of x * gain with the lm_head row of the slot's
// own token, the two sums the logit score (Sec. 3.1) needs from this tile.
// The warp's rows are consecutive and its valid rows a prefix of them.
template <int TBN>
CC_DEV void logit_partials(const GemmParams &p, uint32_t tacc, int grow, bool valid, int nt,
                           int tile_n0, float *stage) {
  const int lane = threadIdx.x & 31, cq = (lane & 7) * 4;
  const int nv = __popc(__ballot_sync(0xFFFFFFFFu, valid));
  const int grow0 = __shfl_sync(0xFFFFFFFFu, grow, 0);
  int tok = valid ? p.tokens[grow] : 0;
  if (tok < 0 || tok >= p.vocab) tok = 0;   // reported by the combine
  int tok_i[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) tok_i[i] = __shfl_sync(0xFFFFFFFFu, tok, 4 * i + (lane >> 3));
  float ss[8], z[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) ss[i] = z[i] = 0.f;
#pragma unroll 1
  for (int c = 0; c < TBN / 32; ++c) {
    uint32_t r[32];
    tmem_ld32(tacc + c * 32, r);
    tmem_ld_wait();
    const int col = tile_n0 + c * 32;
    if (col >= p.N) continue;   // warp-uniform
    stage_chunk(stage, r, lane);
    const uint2 g = *reinterpret_cast<const uint2 *>(p.head_gain + col + cq);
    const float g4[4] = {bf16_lo(g.x), bf16_hi(g.x), bf16_lo(g.y), bf16_hi(g.y)};
    float4 hv[8];
    uint2 wv[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {   // every load first
      const int rr = 4 * i + (lane >> 3);
      hv[i] = make_float4(0.f, 0.f, 0.f, 0.f);
      wv[i] = make_uint2(0u, 0u);
      if (rr >= nv) continue;
      hv[i] = *reinterpret_cast<const float4 *>(
          reinterpret_cast<const float *>(p.out) + (size_t)(grow0 + rr) * p.ldo + col + cq);
      wv[i] = *reinterpret_cast<const uint2 *>(p.head_w + (size_t)tok_i[i] * p.N + col + cq);
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int rr = 4 * i + (lane >> 3);
      const float4 a = *reinterpret_cast<const float4 *>(stage + rr * kStageLd + cq);
      const float x[4] = {a.x + hv[i].x, a.y + hv[i].y, a.z + hv[i].z, a.w + hv[i].w};
      const float w4[4] = {bf16_lo(wv[i].x), bf16_hi(wv[i].x), bf16_lo(wv[i].y), bf16_hi(wv[i].y)};
#pragma unroll
      for (int k = 0; k < 4; ++k) {   // rows past nv add zeros and are never written
        ss[i] = fmaf(x[k], x[k], ss[i]);
        z[i] = fmaf(x[k] * g4[k], w4[k], z[i]);
      }
    }
    __syncwarp();   // the staging tile is rewritten by the next chunk
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const float a = row8_sum(ss[i]), b = row8_sum(z[i]);
    const int rr = 4 * i + (lane >> 3);
    if ((lane & 7) == 0 && rr < nv)
      p.head_part[(size_t)(grow0 + rr) * p.n_tiles + nt] = make_float2(a, b);
  }
}

// fp32 outputs (EPI_F32, EPI_RESID_*), through the staging tile: out = acc
// (+ bf16 resid, or += for RESID_F32); with norm_out (last K split) also
// bf16(out * norm_gain) (and the lo part; fp16 instead with out_f16) and the
// tile's partial sum of out^2.
template <int EPI, int TBN>
CC_DEV void f32_epilogue(const GemmParams &p, uint32_t tacc, int grow, bool valid, int nt,
                         int tile_n0, bool last, float *stage) {
  const int lane = threadIdx.x & 31, cq = (lane & 7) * 4;
  const int nv = __popc(__ballot_sync(0xFFFFFFFFu, valid));
  const int grow0 = __shfl_sync(0xFFFFFFFFu, grow, 0);
  const bool nrm = (EPI == EPI_RESID_BF16 || EPI == EPI_RESID_F32) && p.norm_out && last;
  float ss[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) ss[i] = 0.f;
#pragma unroll 1
  for (int c = 0; c < TBN / 32; ++c) {
    uint32_t r[32];
    tmem_ld32(tacc + c * 32, r);
    tmem_ld_wait();
    const int col = tile_n0 + c * 32;
    if (col >= p.N) continue;   // warp-uniform
    stage_chunk(stage, r, lane);
    float g4[4] = {0.f, 0.f, 0.f, 0.f};
    if (nrm) {
      const uint2 g = *reinterpret_cast<const uint2 *>(p.norm_gain + col + cq);
      g4[0] = bf16_lo(g.x); g4[1] = bf16_hi(g.x); g4[2] = bf16_lo(g.y); g4[3] = bf16_hi(g.y);
    }
    // all eight rows' loads first (the stores below could alias them, so the
    // compiler would not hoist them), then the arithmetic and the stores
    float4 a[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int rr = 4 * i + (lane >> 3);
      a[i] = *reinterpret_cast<const float4 *>(stage + rr * kStageLd + cq);
      if (rr >= nv) continue;
      const size_t row = (size_t)(grow0 + rr);
      if constexpr (EPI == EPI_RESID_BF16) {
        const uint2 h = *reinterpret_cast<const uint2 *>(
            reinterpret_cast<const __nv_bfloat16 *>(p.resid) + row * p.ld_resid + col + cq);
        a[i].x += bf16_lo(h.x); a[i].y += bf16_hi(h.x); a[i].z += bf16_lo(h.y); a[i].w += bf16_hi(h.y);
      } else if constexpr (EPI == EPI_RESID_F32 || EPI == EPI_RESID_LOGIT) {
        const float4 h = *reinterpret_cast<const float4 *>(
            reinterpret_cast<const float *>(p.out) + row * p.ldo + col + cq);
        a[i].x += h.x; a[i].y += h.y; a[i].z += h.z; a[i].w += h.w;
      }
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int rr = 4 * i + (lane >> 3);
      if (rr >= nv) continue;
      const size_t row = (size_t)(grow0 + rr);
      *reinterpret_cast<float4 *>(reinterpret_cast<float *>(p.out) + row * p.ldo + col + cq) = a[i];
      if (nrm) {
        ss[i] = fmaf(a[i].x, a[i].x, ss[i]);
        ss[i] = fmaf(a[i].y, a[i].y, ss[i]);
        ss[i] = fmaf(a[i].z, a[i].z, ss[i]);
        ss[i] = fmaf(a[i].w, a[i].w, ss[i]);
        const float y0 = a[i].x * g4[0], y1 = a[i].y * g4[1], y2 = a[i].z * g4[2],
                    y3 = a[i].w * g4[3];
        bool over = false;
        const uint32_t h0 = pack_act2(y0, y1, p.out_f16, over),
                       h1 = pack_act2(y2, y3, p.out_f16, over);
        if (over) set_status(p.status, CC_ERR_RANGE);
        __nv_bfloat16 *dn = p.norm_out + row * p.ld_norm + col + cq;
        *reinterpret_cast<uint2 *>(dn) = make_uint2(h0, h1);
        if (p.norm_split)   // lo = y * gain - hi, at column offset N
          *reinterpret_cast<uint2 *>(dn + p.N) =
              make_uint2(pack_bf16x2(y0 - bf16_lo(h0), y1 - bf16_hi(h0)),
                         pack_bf16x2(y2 - bf16_lo(h1), y3 - bf16_hi(h1)));
      }
    }
    __syncwarp();   // the staging tile is rewritten by the next chunk
  }
  if (nrm) {
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float v = row8_sum(ss[i]);
      const int rr = 4 * i + (lane >> 3);
      if ((lane & 7) == 0 && rr < nv) p.ss_part[(size_t)(grow0 + rr) * p.n_tiles + nt] = v;
    }
  }
}

template <int EPI, int TBN>
CC_DEV void epilogue_tile(const GemmParams &p, uint32_t tacc, int grow, bool valid, int nt,
                          int tile_n0, bool last, float *stage) {
  if constexpr (EPI == EPI_RESID_LOGIT) {
    if (last) {
      logit_partials<TBN>(p, tacc, grow, valid, nt, tile_n0, stage);
      return;
    }
  }
  if constexpr (EPI == EPI_F32 || EPI == EPI_RESID_BF16 || EPI == EPI_RESID_F32 ||
                EPI == EPI_RESID_LOGIT) {
    f32_epilogue<EPI, TBN>(p, tacc, grow, valid, nt, tile_n0, last, stage);
  } else if constexpr (EPI == EPI_QROPE) {   // kv_fp8: the K rows of an e4m3 cache
    const long long orow = p.kv_dest ? cache_row(p, grow, valid) : grow;
    const bool hm = p.kv_dest && p.pg.head_major;
    if (p.kv_fp8)
      rope_store<TBN, true>(p, tacc, grow, orow, valid, p.out, p.ldo, p.bias, tile_n0, p.N,
                            p.k_qscale, hm);
    else   // with row_ss: the query projection of unnormalised rows (x * gain)
      rope_store<TBN>(p, tacc, grow, orow, valid, p.out, p.ldo, p.bias, tile_n0, p.N, 1.f, hm,
                      p.out_split ? p.N : 0, row_rms_scale(p, grow, valid));
  } else if constexpr (EPI == EPI_BF16) {    // kv_fp8: the V rows of an e4m3 cache
    const long long orow = p.kv_dest ? cache_row(p, grow, valid) : grow;
    const bool hm = p.kv_dest && p.pg.head_major;
    if (p.kv_fp8)
      plain_store<TBN, true>(p, tacc, grow, orow, valid, p.out, p.ldo, p.bias, tile_n0, p.N,
                             p.v_qscale, hm);
    else
      plain_store<TBN>(p, tacc, grow, orow, valid, p.out, p.ldo, p.bias, tile_n0, p.N, 1.f, hm);
  } else if constexpr (EPI == EPI_QKV) {
    // fused projections: column tiles [0, nq) are Q, [nq, nq+nk) K, the rest V (cache rows)
    const int nq = p.n_q_tiles, nk = p.n_k_tiles;
    const long long crow = nt < nq ? grow : cache_row(p, grow, valid);
    const bool hm = p.pg.head_major != 0;   // the K and V parts
    if (nt < nq)
      rope_store<TBN>(p, tacc, grow, grow, valid, p.out, p.ldo, p.bias, nt * TBN, nq * TBN);
    else if (nt < nq + nk && p.kv_fp8)
      rope_store<TBN, true>(p, tacc, grow, crow, valid, p.out_k, p.ldo_kv, p.bias_k,
                            (nt - nq) * TBN, nk * TBN, p.k_qscale, hm);
    else if (nt < nq + nk)
      rope_store<TBN>(p, tacc, grow, crow, valid, p.out_k, p.ldo_kv, p.bias_k, (nt - nq) * TBN,
                      nk * TBN, 1.f, hm);
    else if (p.kv_fp8)
      plain_store<TBN, true>(p, tacc, grow, crow, valid, p.out_v, p.ldo_kv, p.bias_v,
                             (nt - nq - nk) * TBN, nk * TBN, p.v_qscale, hm);
    else
      plain_store<TBN>(p, tacc, grow, crow, valid, p.out_v, p.ldo_kv, p.bias_v,
                       (nt - nq - nk) * TBN, nk * TBN, 1.f, hm);
  } else if constexpr (EPI == EPI_SWIGLU) {
    // columns [0,128) = gate rows nt*128.., [128,256) = up rows nt*128..
    __nv_bfloat16 *out = reinterpret_cast<__nv_bfloat16 *>(p.out) + (size_t)grow * p.ldo;
    const float rs = row_rms_scale(p, grow, valid);   // row_ss: A rows unnormalised
#pragma unroll 1
    for (int c0 = 0; c0 < 128; c0 += 32) {
      uint32_t g[32], u[32];
      tmem_ld32(tacc + c0, g);
      tmem_ld32(tacc + 128 + c0, u);
      tmem_ld_wait();
      int col = nt * 128 + c0;
      if (!valid || col >= p.N) continue;
      float y[32];
#pragma unroll
      for (int k = 0; k < 32; ++k)
        y[k] = silu(__uint_as_float(g[k]) * rs) * (__uint_as_float(u[k]) * rs);
      uint32_t o[16];
      bool over = false;
#pragma unroll
      for (int k = 0; k < 32; k += 2) o[k / 2] = pack_act2(y[k], y[k + 1], p.out_f16, over);
      if (over) set_status(p.status, CC_ERR_RANGE);
      uint4 *d = reinterpret_cast<uint4 *>(out + col);
#pragma unroll
      for (int v = 0; v < 4; ++v) d[v] = make_uint4(o[v * 4], o[v * 4 + 1], o[v * 4 + 2], o[v * 4 + 3]);
      if (p.out_split) {   // lo = bf16(y - hi)
        uint32_t lo[16];
#pragma unroll
        for (int k = 0; k < 32; k += 2)
          lo[k / 2] = pack_bf16x2(y[k] - bf16_lo(o[k / 2]), y[k + 1] - bf16_hi(o[k / 2]));
        uint4 *dl = reinterpret_cast<uint4 *>(out + p.N + col);
#pragma unroll
        for (int v = 0; v < 4; ++v)
          dl[v] = make_uint4(lo[v * 4], lo[v * 4 + 1], lo[v * 4 + 2], lo[v * 4 + 3]);
      }
    }
  } else if constexpr (EPI == EPI_LSE) {
    // per row: (max, sum exp(z - max)) over this tile's vocab columns, and the
    // target logit when the row's token falls in the tile.
    const int tok = valid ? p.tokens[grow] : -1;
    float m = -INFINITY, s = 0.f, zt = 0.f;
    bool has_t = false;
#pragma unroll 1
    for (int c = 0; c < TBN / 32; ++c) {
      uint32_t r[32];
      tmem_ld32(tacc + c * 32, r);
      tmem_ld_wait();
      const int col = tile_n0 + c * 32;
      float cm = -INFINITY;
#pragma unroll
      for (int k = 0; k < 32; ++k)
        if (col + k < p.N) cm = fmaxf(cm, __uint_as_float(r[k]));
      if (cm == -INFINITY) continue;
      if (cm > m) {
        s *= __expf(m - cm);
        m = cm;
      }
#pragma unroll
      for (int k = 0; k < 32; ++k)
        if (col + k < p.N) s += __expf(__uint_as_float(r[k]) - m);
      if (tok >= col && tok < col + 32) {
#pragma unroll
        for (int k = 0; k < 32; ++k)
          if (k == tok - col) zt = __uint_as_float(r[k]);
        has_t = true;
      }
    }
    if (valid) {
      reinterpret_cast<float2 *>(p.out)[(size_t)grow * p.ldo + nt] = make_float2(m, s);
      if (has_t) p.z_target[grow] = zt;
    }
  } else if constexpr (EPI == EPI_ARGMAX) {
    // the tile's largest logit and its first column (NaN never wins)
    float m = -INFINITY;
    int mi = -1;
#pragma unroll 1
    for (int c = 0; c < TBN / 32; ++c) {
      uint32_t r[32];
      tmem_ld32(tacc + c * 32, r);
      tmem_ld_wait();
      const int col = tile_n0 + c * 32;
#pragma unroll
      for (int k = 0; k < 32; ++k) {
        const float v = __uint_as_float(r[k]);
        if (col + k < p.N && v > m) {
          m = v;
          mi = col + k;
        }
      }
    }
    if (valid)
      reinterpret_cast<float2 *>(p.out)[(size_t)(grow / p.cap) * p.ldo + nt] =
          make_float2(m, __int_as_float(mi));
  }
}

// Tile t -> (row tile m, column tile n) in grouped order: consecutive tiles
// stay inside one group of `group` resident tiles of one operand while the
// other operand's tiles stream past (see GemmParams::raster).
CC_DEV void tile_coords(const GemmParams &p, int t, int num_m, int &m, int &n) {
  const int num_n = p.n_tiles;
  if (p.raster == 0) {   // resident column tiles, rows stream
    const int per = num_m * p.group;
    const int g = t / per, r = t - g * per;
    const int gn = min(p.group, num_n - g * p.group);
    m = r / gn;
    n = g * p.group + (r - m * gn);
  } else {               // resident row tiles, columns stream
    const int per = num_n * p.group;
    const int g = t / per, r = t - g * per;
    const int gm = min(p.group, num_m - g * p.group);
    n = r / gm;
    m = g * p.group + (r - n * gm);
  }
}

// One CTA per SM (PAIR false) or a CTA pair per two SMs (PAIR true, a
// cluster of two), persistent over the output tiles.  A pair computes
// 256-row tiles: CTA r holds row tile 2 mu + r of row unit mu (two
// consecutive 128-row tiles, which may belong to different sequences) and B rows
// [r TBN/2, (r+1) TBN/2) of the column tile; CTA 0 issues the pair's
// products into both tensor memories and its commits release the stages
// and accumulators of both CTAs.  Both CTAs' loads of a stage complete on
// CTA 0's stage barrier (CTA 0 arms it with the bytes of both), and CTA 1's
// epilogue warps release an accumulator by arriving on CTA 0's barrier.
// (A relay thread in CTA 1 that waited for its own stage barrier and then
// arrived on CTA 0's measured 3.4x slower on the gate/up shape: the
// hand-over latency sat on every stage.)  K splits run on single CTAs only.
template <int EPI, int TBN, bool PAIR>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                const __grid_constant__ CUtensorMap tmB2, const __grid_constant__ CUtensorMap tmB3,
                const __grid_constant__ GemmParams p) {
  constexpr int kSt = (int)stages(PAIR);
  // CTA pairs wait and commit once per two 64-deep k-blocks (a barrier stage
  // = two consecutive ring slots, 64 KB of the pair's operands): per product
  // issued, half the barrier waits, expect-tx arms and commits.  Measured on
  // the Llama-3-8B 16k step (fp16 operands): gate/up 2.24 -> 2.15 ms per
  // launch at a lower clock (1620 -> 1575 MHz), the step 185.7 -> 183.6 ms.
  constexpr int KB2 = PAIR ? 2 : 1;   // k-blocks per barrier stage
  constexpr int kSS = kSt / KB2;      // barrier stages
  static_assert(kSt % KB2 == 0, "whole barrier stages");
  constexpr int TB_BYTES = TBN * BK * 2;                  // B tile of one product
  constexpr int SB = PAIR ? TB_BYTES / 2 : TB_BYTES;       // B stage: this CTA's share
  static_assert(!PAIR || TBN == BN, "CTA pairs use 256-column tiles");
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                              ~uintptr_t(1023));
  uint8_t *sA = smem;
  uint8_t *sB = smem + kSt * A_BYTES;
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + ring_bytes(PAIR));
  uint64_t *empty = full + kSt;
  uint64_t *tfull = empty + kSt;
  uint64_t *tempty = tfull + 2;
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(tempty + 2);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);
  int *prefix = reinterpret_cast<int *>(smem + ring_bytes(PAIR) + 256);
  float *stage_all = reinterpret_cast<float *>(smem + ring_bytes(PAIR) + 256 + kPrefixBytes);
  __shared__ int split_ok;   // K splits: the previous split of the tile has published

  // a pair kernel launched without its cluster of two has no partner for
  // the pair instructions: every CTA reports it and leaves before any
  if (PAIR && cluster_nctarank() != 2) {
    if (threadIdx.x == 0) set_status(p.status, CC_ERR_DEVICE_ARG);
    return;
  }
  const uint32_t rank = PAIR ? cluster_ctarank() : 0;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kSt; ++s) {
      mbar_init(&full[s], 1);   // CTA 1 of a pair leaves its own unused
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], PAIR ? 8 : 4);   // the epilogue warps (of both CTAs)
    }
    *abort_flag = 0;
    build_tile_prefix(p.seq_len, p.row_lo, p.batch, p.cap, BM, prefix, p.status);
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    if (EPI == EPI_SWIGLU || EPI == EPI_QKV) tma_prefetch_desc(&tmB2);
    if (EPI == EPI_QKV) tma_prefetch_desc(&tmB3);
  }
  if (warp == 1) {
    if constexpr (PAIR) tmem_alloc_pair(tmem_slot, 512);
    else tmem_alloc(tmem_slot, 512);
  }
  tc_fence_before();
  __syncthreads();
  if constexpr (PAIR) cluster_sync();   // both CTAs' barriers exist before any remote arrival
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int num_m = prefix[p.batch];
  const int num_mu = PAIR ? (num_m + 1) / 2 : num_m;   // row units: tiles or tile pairs
  const int total = num_mu * p.n_tiles;
  const int nk = (p.K + BK - 1) / BK;           // k-blocks of one operand pass
  const int nk_total = p.a_split ? 2 * nk : nk;  // split A: the hi pass, then the lo pass
  // Work item = (tile, K split): the splits of a tile are consecutive items.
  const int S = (!PAIR && (EPI == EPI_RESID_F32 || EPI == EPI_RESID_LOGIT) && p.k_splits > 1)
                    ? p.k_splits
                    : 1;
  const int total_items = total * S;
  const int unit0 = PAIR ? (int)(blockIdx.x >> 1) : (int)blockIdx.x;
  const int n_units = PAIR ? (int)(gridDim.x >> 1) : (int)gridDim.x;
  // row tile of this CTA in row unit u (-1: past the last tile, the second
  // CTA of an odd pair: it loads its B share only and stores nothing)
  auto row_tile = [&](int u) { const int mt = PAIR ? 2 * u + (int)rank : u; return mt < num_m ? mt : -1; };

  if (warp == 0) {
    if (lane == 0) {  // ---------------- TMA producer
      // L2 policies: the resident operand evict-last, the streamed one
      // evict-first; CTA pairs keep both evict-last (measured at the Llama-3-8B
      // 16k launches: evict-first A made the pairs re-read it from DRAM,
      // gate/up 4.3 -> 1.7 GB and 1.98 -> 1.92 ms, down 5.5 -> 3.5 GB and
      // 1.09 -> 1.05 ms)
      const uint64_t keep = make_policy_evict_last(), stream = make_policy_evict_first();
      const uint64_t pol_a = PAIR || p.raster == 1 ? keep : stream;
      const uint64_t pol_b = PAIR || p.raster == 0 ? keep : stream;
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int item = unit0; ok && item < total_items; item += n_units) {
        const int tile = item / S, split = item - tile * S;
        int mu, nt;
        tile_coords(p, tile, num_mu, mu, nt);
        const int mt = row_tile(mu);
        int row0 = 0;
        if (mt >= 0) {
          const int b = find_seq(prefix, p.batch, mt);
          row0 = b * p.cap + (p.row_lo ? p.row_lo[b] : 0) + (mt - prefix[b]) * BM;
        }
        const int kb0 = split * nk_total / S, kb1 = (split + 1) * nk_total / S;
        // a pair's second row tile exists (CTA 0 counts its A bytes)
        const bool a1 = PAIR && 2 * mu + 1 < num_m;
        for (int kbs = kb0; kbs < kb1; kbs += KB2) {
          const int nb = min(KB2, kb1 - kbs);
          if (!(ok = mbar_wait(&empty[stage], phase ^ 1, abort_flag, p.status))) break;
          if (!PAIR) mbar_arrive_expect_tx(&full[stage], nb * (A_BYTES + TB_BYTES));
          else if (rank == 0) mbar_arrive_expect_tx(&full[stage], nb * ((a1 ? 2 : 1) * A_BYTES + TB_BYTES));
          const uint32_t bar_cl = PAIR ? cluster_addr(&full[stage], 0) : 0;
          auto load = [&](uint8_t *dst, const CUtensorMap *m, int c0, int c1, uint64_t pol) {
            if constexpr (PAIR) tma_load_2d_pair_hint(dst, m, bar_cl, c0, c1, pol);
            else tma_load_2d_hint(dst, m, &full[stage], c0, c1, pol);
          };
          for (int j = 0; j < nb; ++j) {   // the stage's k-blocks, one ring slot each
            const int kb = kbs + j, slot = stage * KB2 + j;
            // A column block kb of [hi | lo] (hi and lo halves are K apart), B block kb mod nk
            const int ka = kb < nk ? kb * BK : p.K + (kb - nk) * BK;
            const int kw = (kb < nk ? kb : kb - nk) * BK;
            if (mt >= 0) load(sA + slot * A_BYTES, &tmA, ka, row0, pol_a);
            uint8_t *sb = sB + slot * SB;
            if constexpr (EPI == EPI_SWIGLU) {   // gate rows, then up rows (CTA 0: gate, CTA 1: up)
              if (!PAIR || rank == 0) load(sb, &tmB, kw, nt * 128, pol_b);
              if (!PAIR || rank == 1) load(PAIR ? sb : sb + TB_BYTES / 2, &tmB2, kw, nt * 128, pol_b);
            } else if constexpr (EPI == EPI_QKV) {
              const int nq = p.n_q_tiles, nkt = p.n_k_tiles;
              const CUtensorMap *m = nt < nq ? &tmB : (nt < nq + nkt ? &tmB2 : &tmB3);
              const int r0 = (nt < nq ? nt : (nt < nq + nkt ? nt - nq : nt - nq - nkt)) * TBN;
              load(sb, m, kw, r0 + (int)rank * (TBN / 2), pol_b);
            } else {
              load(sb, &tmB, kw, nt * TBN + (int)rank * (TBN / 2), pol_b);
            }
          }
          if (++stage == kSS) { stage = 0; phase ^= 1; }
        }
      }
      if (PAIR && ok) {
        // every stage's last release (a commit of CTA 0) has landed before
        // the CTA may leave
        for (int i = 0; i < kSS; ++i) {
          if (!mbar_wait(&empty[stage], phase ^ 1, abort_flag, p.status)) break;
          if (++stage == kSS) { stage = 0; phase ^= 1; }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) {  // ---------------- MMA issuer (CTA 0 of a pair)
      const uint32_t idesc = p.ab_f16 ? make_idesc_f16(PAIR ? 2 * BM : BM, TBN, 0, 0)
                                      : make_idesc_bf16(PAIR ? 2 * BM : BM, TBN, 0, 0);
      const uint64_t a_desc0 = make_sdesc_sw128(smem_u32(sA), 16, 1024);
      const uint64_t b_desc0 = make_sdesc_sw128(smem_u32(sB), 16, 1024);
      int stage = 0, acc = 0;
      uint32_t phase = 0, acc_phase = 0;
      for (int item = unit0; item < total_items; item += n_units) {
        const int split = item % S;
        const int kb0 = split * nk_total / S, kb1 = (split + 1) * nk_total / S;
        if (!mbar_wait<PAIR>(&tempty[acc], acc_phase ^ 1, abort_flag, p.status)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * TBN;
        for (int kbs = kb0; kbs < kb1; kbs += KB2) {
          const int nb = min(KB2, kb1 - kbs);
          if (!mbar_wait<PAIR>(&full[stage], phase, abort_flag, p.status)) goto mma_done;
          tc_fence_after();
          for (int j = 0; j < nb; ++j) {
            const int kb = kbs + j, slot = stage * KB2 + j;
            // descriptors of this stage; a K step of 16 columns advances the
            // start-address field by 32 bytes (+2 in 16-byte units)
            const uint64_t ad = a_desc0 + (uint64_t)(slot * (A_BYTES >> 4));
            const uint64_t bd = b_desc0 + (uint64_t)(slot * (SB >> 4));
#pragma unroll
            for (int k = 0; k < BK / 16; ++k) {
              const uint32_t accum = (kb != kb0 || k != 0) ? 1u : 0u;
              if constexpr (PAIR) umma_ss_pair(d_tmem, ad + 2 * k, bd + 2 * k, idesc, accum);
              else umma_ss(d_tmem, ad + 2 * k, bd + 2 * k, idesc, accum);
            }
          }
          if constexpr (PAIR) umma_commit_pair(&empty[stage], 0x3);
          else umma_commit(&empty[stage]);
          if (++stage == kSS) { stage = 0; phase ^= 1; }
        }
        if constexpr (PAIR) umma_commit_pair(&tfull[acc], 0x3);
        else umma_commit(&tfull[acc]);
        if (++acc == 2) { acc = 0; acc_phase ^= 1; }
      }
    mma_done:;
    }
  } else {  // ------------------------------ epilogue warps 2..5
    const int q = warp & 3;        // TMEM lane quarter this warp may access
    const int r = q * 32 + lane;   // accumulator row of this thread
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int item = unit0; item < total_items; item += n_units) {
      const int tile = item / S, split = item - tile * S;
      int mu, nt;
      tile_coords(p, tile, num_mu, mu, nt);
      const int mt = row_tile(mu);
      bool valid = false;
      int grow = 0;
      if (mt >= 0) {
        const int b = find_seq(prefix, p.batch, mt);
        const int i = (p.row_lo ? p.row_lo[b] : 0) + (mt - prefix[b]) * BM + r;
        valid = i < (p.seq_len ? p.seq_len[b] : p.cap);
        grow = b * p.cap + i;
      }
      if (!mbar_wait(&tfull[acc], acc_phase, abort_flag, p.status)) break;
      tc_fence_after();
      const uint32_t tacc = tmem_base + acc * TBN + (uint32_t(q * 32) << 16);
      // K splits add into out in split order (deterministic sums): split s
      // waits until split s-1 of the tile has published epoch * 16 + s.
      // Split s-1 is a lower work item, and every CTA takes its items in
      // increasing order, so the wait always ends (bounded all the same).
      bool add = mt >= 0;
      if (S > 1) {
        if (warp == 2 && lane == 0)
          split_ok = split == 0 || wait_value(&p.split_flags[tile], p.epoch * 16u + split, p.status);
        named_barrier_sync(1, 128);
        add = split_ok != 0;   // a wait that gave up (status set) skips this split's add
      }
      if (add)
        epilogue_tile<EPI, TBN>(p, tacc, grow, valid, nt, nt * TBN, split == S - 1,
                                stage_all + q * 32 * kStageLd);
      tc_fence_before();
      if (S > 1) {
        named_barrier_sync(1, 128);
        if (warp == 2 && lane == 0) {
          __threadfence();
          st_release_u32(&p.split_flags[tile], p.epoch * 16u + split + 1);
        }
      }
      __syncwarp();
      if (lane == 0) {
        if (PAIR && rank == 1) mbar_arrive_cluster(cluster_addr(&tempty[acc], 0));
        else mbar_arrive(&tempty[acc]);
      }
      if (++acc == 2) { acc = 0; acc_phase ^= 1; }
    }
  }

  tc_fence_before();
  __syncthreads();
  if constexpr (PAIR) cluster_sync();   // the partner is done with this CTA's memories
  if (*abort_flag) __nanosleep(1000000);   // let copies still in flight land
  if (warp == 1) {
    tc_fence_after();
    if constexpr (PAIR) tmem_dealloc_pair(tmem_base, 512);
    else tmem_dealloc(tmem_base, 512);
  }
}

template <int EPI, int TBN, bool PAIR>
cudaError_t launch_t(const CUtensorMap &a, const CUtensorMap &b, const CUtensorMap &b2,
                     const CUtensorMap &b3, const GemmParams &p, int grid, cudaStream_t stream) {
  auto kern = gemm_kernel<EPI, TBN, PAIR>;
  static bool attr_set[64] = {};
  static int max_pairs[64] = {};   // co-resident CTA pairs (cluster occupancy)
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 64 && !attr_set[dev]) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem_bytes(PAIR));
    if (e != cudaSuccess) return e;
    attr_set[dev] = true;
  }
  if constexpr (!PAIR) {
    kern<<<grid, kThreads, smem_bytes(false), stream>>>(a, b, b2, b3, p);
    return cudaGetLastError();
  } else {
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2 * (unsigned)std::max(grid / 2, 1));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem_bytes(true);
    cfg.stream = stream;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int pairs = grid / 2;
    if (dev < 64) {
      if (max_pairs[dev] == 0) {
        int n = 0;
        cudaError_t e = cudaOccupancyMaxActiveClusters(&n, kern, &cfg);
        if (e != cudaSuccess) return e;
        max_pairs[dev] = std::max(n, 1);
      }
      pairs = std::min(pairs, max_pairs[dev]);
    }
    cfg.gridDim = dim3(2 * (unsigned)std::max(pairs, 1));
    return cudaLaunchKernelEx(&cfg, kern, a, b, b2, b3, p);
  }
}

// SwiGLU (gate and up halves), LSE and the fused q/k/v projections always
// use 256-wide tiles; the others take p.block_n (128 or 256).  p.pair: CTA
// pairs (256-wide tiles only; greedy decoding's argmax never pairs).
template <int EPI>
cudaError_t launch(const CUtensorMap &a, const CUtensorMap &b, const CUtensorMap &b2,
                   const CUtensorMap &b3, const GemmParams &p, int grid, cudaStream_t stream) {
  constexpr bool kWide = EPI == EPI_SWIGLU || EPI == EPI_LSE || EPI == EPI_QKV;
  if constexpr (EPI != EPI_ARGMAX) {
    if (p.pair && (kWide || p.block_n == BN)) return launch_t<EPI, BN, true>(a, b, b2, b3, p, grid, stream);
  }
  if (p.pair) return cudaErrorInvalidValue;
  if constexpr (kWide) {
    return launch_t<EPI, BN, false>(a, b, b2, b3, p, grid, stream);
  } else {
    if (p.block_n == 128) return launch_t<EPI, 128, false>(a, b, b2, b3, p, grid, stream);
    return launch_t<EPI, BN, false>(a, b, b2, b3, p, grid, stream);
  }
}

}  // namespace

int gemm_block_n(int epi) { return epi == EPI_SWIGLU ? 128 : BN; }
int gemm_max_batch() { return kMaxBatch; }

cudaError_t launch_gemm(int epi, const CUtensorMap &a, const CUtensorMap &b, const CUtensorMap &b2,
                        const CUtensorMap &b3, const GemmParams &p, int grid, cudaStream_t stream) {
  switch (epi) {
    case EPI_F32: return launch<EPI_F32>(a, b, b2, b3, p, grid, stream);
    case EPI_QROPE: return launch<EPI_QROPE>(a, b, b2, b3, p, grid, stream);
    case EPI_RESID_BF16: return launch<EPI_RESID_BF16>(a, b, b2, b3, p, grid, stream);
    case EPI_RESID_F32: return launch<EPI_RESID_F32>(a, b, b2, b3, p, grid, stream);
    case EPI_SWIGLU: return launch<EPI_SWIGLU>(a, b, b2, b3, p, grid, stream);
    case EPI_LSE: return launch<EPI_LSE>(a, b, b2, b3, p, grid, stream);
    case EPI_BF16: return launch<EPI_BF16>(a, b, b2, b3, p, grid, stream);
    case EPI_QKV: return launch<EPI_QKV>(a, b, b2, b3, p, grid, stream);
    case EPI_ARGMAX: return launch<EPI_ARGMAX>(a, b, b2, b3, p, grid, stream);
    case EPI_RESID_LOGIT: return launch<EPI_RESID_LOGIT>(a, b, b2, b3, p, grid, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace cc
