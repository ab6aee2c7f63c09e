// keyattn.cu -- attention received by each cached key when cached keys act
// as proxy queries: the paper's importance and heavy-hitter (H2O) comparison
// scorers (Sec. 4) on the same keep-set path as the counter-causal score.
//
// For one layer's K cache and KV head g of sequence b, query slot i in
// [q_lo, n) attends keys j <= i with weights softmax_j(K[i] . K[j] / sqrt(dh)).
// Two sweeps, both S = X Y^T on tcgen05 (M = N = 128, K = dh, fp32 in TMEM):
//   sweep 0: rows = proxy-query slots, stream = key tiles 0 .. the block's
//            last row; per row the log2-sum-exp lse2[i] (online max/sum).
//   sweep 1: rows = key slots, stream = proxy-query tiles from the block's
//            first key (or q_lo) to n-1, each with its 128 lse2 values; per
//            row (key) the sum of 2^(s * c - lse2[i]) over its queries
//            i >= max(j, q_lo): the column sum is a row sum of the
//            transposed product, so each thread adds its own key's weights.
// Per-head sums go to part[b][g][j]; a finishing kernel adds the heads in a
// fixed order (deterministic, no atomics).
//
//   warps 0..3  rows (one per thread): S from TMEM, mask, reduce
//   warp 4      TMA producer (row tile once; stream tiles, 2 stages; sweep
//               1 also bulk-copies the tile's lse2 values)
//   warp 5      TMEM owner + tcgen05.mma issuer; S double-buffered in TMEM
//               (no P V product here, so S of tile t+1 never waits on t)
#include "keyattn.cuh"

namespace cc {

namespace {

constexpr int KT = 128;         // slots per tile
constexpr int KST = 2;          // stream stages
constexpr int kThreads = 192;   // 4 row warps, producer, MMA

template <int DH>
struct KaSmem {
  static constexpr int NH = DH / 64;                  // 64-column (128-byte) halves
  static constexpr int TILE = NH * KT * 128;          // one 128-slot x DH tile
  static constexpr int OFF_ROW = 0;
  static constexpr int OFF_STR = OFF_ROW + TILE;
  static constexpr int OFF_LSE = OFF_STR + KST * TILE;   // [KST][KT] floats (sweep 1)
  static constexpr int OFF_BAR = OFF_LSE + KST * KT * 4;
  static constexpr int BYTES = OFF_BAR + 128 + 1024;     // barriers + alignment slack
};

CC_DEV float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

template <int DH, int SWEEP>
__global__ void __launch_bounds__(kThreads)
    keyattn_kernel(const __grid_constant__ KeyAttnBatch batch_args) {
  using L = KaSmem<DH>;
  const KeyAttnParams &p = batch_args.p;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                              ~uintptr_t(1023));
  uint64_t *bars = reinterpret_cast<uint64_t *>(smem + L::OFF_BAR);
  uint64_t *row_full = bars;
  uint64_t *str_full = bars + 1;           // [KST]
  uint64_t *str_empty = str_full + KST;    // [KST]
  uint64_t *s_full = str_empty + KST;      // [2]
  uint64_t *s_empty = s_full + 2;          // [2]
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(s_empty + 2);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);
  const float *lse_st = reinterpret_cast<const float *>(smem + L::OFF_LSE);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int per_seq = SWEEP == 0 ? (p.q_span + KT - 1) / KT : (p.cap + KT - 1) / KT;
  const int blk = blockIdx.x % per_seq;
  const int bg = blockIdx.x / per_seq;
  const int g = bg % p.n_kv_heads, b = bg / p.n_kv_heads;
  const int layer = blockIdx.y;
  const CUtensorMap &tmK = batch_args.k[layer];
  const int n = p.seq_len[b];
  int q_lo = p.q_lo ? p.q_lo[b] : (p.recent > 0 ? max(0, n - p.recent) : 0);
  if (n < 0 || n > p.cap || q_lo < 0 || q_lo > n) {
    if (threadIdx.x == 0) set_status(p.status, CC_ERR_DEVICE_ARG);
    return;
  }
  const size_t head_off = (((size_t)layer * p.batch + b) * p.n_kv_heads + g) * p.ld;
  int row0, t_first, t_last;
  if (SWEEP == 0) {   // rows: proxy queries; keys 0 .. the block's last query
    row0 = q_lo + blk * KT;
    if (row0 >= n) return;
    t_first = 0;
    t_last = (min(row0 + KT, n) - 1) / KT;
  } else {            // rows: keys; queries max(row0, q_lo) .. n-1
    row0 = blk * KT;
    if (row0 >= n) return;
    const int first_q = max(row0, q_lo);
    if (first_q >= n) {   // no query sees these keys
      if (threadIdx.x < KT && row0 + (int)threadIdx.x < n) p.part[head_off + row0 + threadIdx.x] = 0.f;
      return;
    }
    t_first = first_q / KT;
    t_last = (n - 1) / KT;
  }
  const int ntiles = t_last - t_first + 1;
  // pool row of the key tile starting at slot i (paged: one page holds it);
  // a bad page reads zeros (a coordinate past the map) and is reported
  auto tile_row = [&](int i) -> int {
    if (p.pg.head_major) return b * p.n_kv_heads + g;   // coordinates (slot, b*Hkv + g)
    const long long r = kv_row(p.pg, p.cap, b, i);
    if (r < 0) {
      set_status(p.status, CC_ERR_DEVICE_ARG);
      return p.kv_rows;
    }
    return (int)r;
  };

  if (threadIdx.x == 0) {
    mbar_init(row_full, 1);
    for (int s = 0; s < KST; ++s) {
      mbar_init(&str_full[s], 1);
      mbar_init(&str_empty[s], SWEEP == 1 ? 1 + 4 : 1);   // sweep 1: row warps read the lse2 stage
    }
    for (int h = 0; h < 2; ++h) {
      mbar_init(&s_full[h], 1);
      mbar_init(&s_empty[h], 4);
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 5) tmem_alloc(tmem_slot, 256);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 4) {
    // -------------------------------------------------------------- producer
    if (lane == 0) {
      tma_prefetch_desc(&tmK);
      mbar_arrive_expect_tx(row_full, L::TILE);
      for (int hh = 0; hh < L::NH; ++hh)
        tma_load_3d(smem + L::OFF_ROW + hh * KT * 128, &tmK, row_full, hh * 64,
                    p.pg.head_major ? row0 : g, tile_row(row0));
      for (int it = 0; it < ntiles; ++it) {
        const int t = t_first + it, s = it % KST;
        const uint32_t ph = (it / KST) & 1;
        if (!mbar_wait(&str_empty[s], ph ^ 1, abort_flag, p.status)) break;
        mbar_arrive_expect_tx(&str_full[s], L::TILE + (SWEEP == 1 ? KT * 4 : 0));
        for (int hh = 0; hh < L::NH; ++hh)
          tma_load_3d(smem + L::OFF_STR + s * L::TILE + hh * KT * 128, &tmK, &str_full[s], hh * 64,
                      p.pg.head_major ? t * KT : g, tile_row(t * KT));
        if (SWEEP == 1)
          bulk_load(smem + L::OFF_LSE + s * KT * 4, p.lse + head_off + (size_t)t * KT, KT * 4,
                    &str_full[s]);
      }
    }
  } else if (warp == 5) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = make_idesc_bf16(128, KT, 0, 0);
      const uint64_t row_desc = make_sdesc_sw128(smem_u32(smem + L::OFF_ROW), 16, 1024);
      const uint64_t str_desc = make_sdesc_sw128(smem_u32(smem + L::OFF_STR), 16, 1024);
      bool ok = mbar_wait(row_full, 0, abort_flag, p.status);
      for (int it = 0; ok && it < ntiles; ++it) {
        const int s = it % KST, buf = it & 1;
        if (!(ok = mbar_wait(&str_full[s], (it / KST) & 1, abort_flag, p.status))) break;
        if (!(ok = mbar_wait(&s_empty[buf], ((it / 2) & 1) ^ 1, abort_flag, p.status))) break;
        tc_fence_after();
        const uint64_t sd = str_desc + (uint64_t)((s * L::TILE) >> 4);
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk) {
          // K step of 16 columns: +32 bytes within a 128-byte row; 64-column
          // halves are KT * 128 bytes apart
          const uint64_t off = (uint64_t)((((kk >> 2) * KT * 128) >> 4) + (kk & 3) * 2);
          umma_ss(tmem + buf * KT, row_desc + off, sd + off, idesc, kk > 0);
        }
        umma_commit(&s_full[buf]);
        umma_commit(&str_empty[s]);
      }
    }
  } else {
    // ------------------------------------------------------------------ rows
    const int r = warp * 32 + lane;
    const int i_row = row0 + r;                 // slot of this row (query or key)
    const uint32_t lane_off = uint32_t(warp * 32) << 16;
    const float c = p.scale_log2;
    float m = -INFINITY, l = 0.f, acc = 0.f;
    bool ok = true;
    for (int it = 0; it < ntiles; ++it) {
      const int buf = it & 1, s = it % KST;
      const int j0 = (t_first + it) * KT;       // first slot of the stream tile
      if (!(ok = mbar_wait(&s_full[buf], (it / 2) & 1, abort_flag, p.status))) break;
      tc_fence_after();
      uint32_t sr[128];
      tmem_ld32(tmem + lane_off + buf * KT + 0, *reinterpret_cast<uint32_t(*)[32]>(&sr[0]));
      tmem_ld32(tmem + lane_off + buf * KT + 32, *reinterpret_cast<uint32_t(*)[32]>(&sr[32]));
      tmem_ld32(tmem + lane_off + buf * KT + 64, *reinterpret_cast<uint32_t(*)[32]>(&sr[64]));
      tmem_ld32(tmem + lane_off + buf * KT + 96, *reinterpret_cast<uint32_t(*)[32]>(&sr[96]));
      tmem_ld_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&s_empty[buf]);   // S copied out: the buffer may be refilled
      if (SWEEP == 0) {
        // key j0 + col kept iff j <= min(i, n - 1)
        const int hi = min(i_row, n - 1) - j0 + 1;
        float mp[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
        for (int col = 0; col < 128; ++col) {
          const float y = col < hi ? __uint_as_float(sr[col]) * c : -INFINITY;
          sr[col] = __float_as_uint(y);
          mp[col & 3] = fmaxf(mp[col & 3], y);
        }
        const float m_new = fmaxf(m, fmaxf(fmaxf(mp[0], mp[1]), fmaxf(mp[2], mp[3])));
        float sum = 0.f;
#pragma unroll
        for (int col = 0; col < 128; ++col) sum += ex2(__uint_as_float(sr[col]) - m_new);
        l = (m == -INFINITY ? 0.f : l * ex2(m - m_new)) + sum;
        m = m_new;
      } else {
        // query j0 + col counted iff max(j, q_lo) <= i < n; the tile's lse2
        // values landed with its stream stage (already complete here)
        if (!(ok = mbar_wait(&str_full[s], (it / KST) & 1, abort_flag, p.status))) break;
        const int lo = max(i_row, q_lo) - j0, hi = n - j0;
        const float *ls = lse_st + s * KT;
        float a2[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int col = 0; col < 128; ++col) {
          const float w = ex2(__uint_as_float(sr[col]) * c - ls[col]);
          a2[col & 3] += (col >= lo && col < hi) ? w : 0.f;
        }
        acc += (a2[0] + a2[1]) + (a2[2] + a2[3]);
        __syncwarp();
        if (lane == 0) mbar_arrive(&str_empty[s]);   // lse2 stage read
      }
    }
    if (ok && i_row < n) {
      if (SWEEP == 0)
        p.lse[head_off + i_row] = m + __log2f(l);
      else
        p.part[head_off + i_row] = acc;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (*abort_flag) __nanosleep(1000000);   // let copies still in flight land
  if (warp == 5) {
    tc_fence_after();
    tmem_dealloc(tmem, 256);
  }
}

// out[b][j] = (accumulate ? out : 0) + sum_g part[b][g][j] (/ Hkv (n - j) when mean)
__global__ void keyattn_finish_kernel(const KeyAttnParams p, float *out, int mean,
                                      int accumulate) {
  const int b = blockIdx.y;
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= p.cap) return;
  const int n = p.seq_len[b];
  float *o = out + (size_t)b * p.cap + j;
  if (n < 0 || n > p.cap || j >= n) {
    if (!accumulate) *o = -INFINITY;
    return;
  }
  float s = 0.f;
  for (int l = 0; l < p.n_layers; ++l)
    for (int g = 0; g < p.n_kv_heads; ++g)
      s += p.part[(((size_t)l * p.batch + b) * p.n_kv_heads + g) * p.ld + j];
  if (mean) s /= (float)p.n_kv_heads * (float)(n - j);
  *o = accumulate ? *o + s : s;
}

// Sliding window: the score of a slot is its original position.
__global__ void recency_kernel(const int32_t *pos, const int32_t *seq_len, int cap, float *scores) {
  const int b = blockIdx.y;
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= cap) return;
  const int n = seq_len[b];
  const size_t i = (size_t)b * cap + j;
  scores[i] = (j < n && n <= cap) ? (float)pos[i] : -INFINITY;
}

// H2O refresh scores: the running total; the `recent` last slots always kept.
__global__ void h2o_scores_kernel(const float *acc, const int32_t *seq_len, int cap, int recent,
                                  float *scores) {
  const int b = blockIdx.y;
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= cap) return;
  const int n = seq_len[b];
  const size_t i = (size_t)b * cap + j;
  if (j >= n || n > cap)
    scores[i] = -INFINITY;
  else
    scores[i] = j >= n - recent ? INFINITY : acc[i];
}

template <int DH>
cudaError_t launch_dh(const KeyAttnBatch &a, cudaStream_t st) {
  const KeyAttnParams &p = a.p;
  static bool attr_set[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 64 && !attr_set[dev]) {
    cudaError_t e = cudaFuncSetAttribute(keyattn_kernel<DH, 0>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, KaSmem<DH>::BYTES);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(keyattn_kernel<DH, 1>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               KaSmem<DH>::BYTES);
    if (e != cudaSuccess) return e;
    attr_set[dev] = true;
  }
  const long long heads = (long long)p.batch * p.n_kv_heads;
  const long long u0 = heads * ((p.q_span + KT - 1) / KT);
  const long long u1 = heads * ((p.cap + KT - 1) / KT);
  if (p.n_layers < 1 || p.n_layers > kKeyAttnMaxLayers) return cudaErrorInvalidValue;
  if (u0 > 0)
    keyattn_kernel<DH, 0><<<dim3((unsigned)u0, p.n_layers), kThreads, KaSmem<DH>::BYTES, st>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (u1 > 0)
    keyattn_kernel<DH, 1><<<dim3((unsigned)u1, p.n_layers), kThreads, KaSmem<DH>::BYTES, st>>>(a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_keyattn(const KeyAttnBatch &a, cudaStream_t st) {
  if (a.p.head_dim == 128) return launch_dh<128>(a, st);
  if (a.p.head_dim == 64) return launch_dh<64>(a, st);
  return cudaErrorInvalidValue;
}

cudaError_t launch_keyattn_finish(const KeyAttnParams &p, float *out, bool mean, bool accumulate,
                                  cudaStream_t st) {
  const dim3 grid((p.cap + 255) / 256, p.batch);
  keyattn_finish_kernel<<<grid, 256, 0, st>>>(p, out, mean ? 1 : 0, accumulate ? 1 : 0);
  return cudaGetLastError();
}

cudaError_t launch_recency_scores(const int32_t *pos, const int32_t *seq_len, int batch, int cap,
                                  float *scores, cudaStream_t st) {
  recency_kernel<<<dim3((cap + 255) / 256, batch), 256, 0, st>>>(pos, seq_len, cap, scores);
  return cudaGetLastError();
}

cudaError_t launch_h2o_scores(const float *acc, const int32_t *seq_len, int batch, int cap,
                              int recent, float *scores, cudaStream_t st) {
  h2o_scores_kernel<<<dim3((cap + 255) / 256, batch), 256, 0, st>>>(acc, seq_len, cap, recent,
                                                                   scores);
  return cudaGetLastError();
}

}  // namespace cc
