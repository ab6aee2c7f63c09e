// gemv.cu -- weight-streaming products of a few rows (decode step): the
// layer products of DoInference for one token per sequence (Sec. 3,
// Algorithm DoInference) and the LM head's greedy choice.
//
// Persistent CTA per SM over a contiguous range of row groups.
//   producer warp:  for each group and each K piece of KS x 256 elements,
//                   2 x KS TMA boxes of 8 weight rows x 256 into the next ring
//                   stage (weights streamed once: L2 evict-first).
//   16 consumer warps: stage the batch rows in shared memory first (bf16;
//                   optionally the RMSNorm of fp32 rows, rounded as the norm
//                   kernel rounds), then warp w takes row w of every stage:
//                   16 bytes per lane against the staged rows, so a group's
//                   16 outputs are the 16 warps' dot products (fixed order).
//   warp 0 also:    the group's epilogue, from a double-buffered result slot
//                   (group barriers: slot full after 16 warp arrivals, slot
//                   free after the epilogue).
// Every wait is bounded (status CC_ERR_TIMEOUT, abort flag for the others).
#include "gemv.cuh"

namespace cc {

namespace {

constexpr int kThreads = (kGemvConsumers + 1) * 32;   // + the producer warp

CC_DEV void unpack8f(const uint4 &v, float *f) {
  f[0] = bf16_lo(v.x); f[1] = bf16_hi(v.x); f[2] = bf16_lo(v.y); f[3] = bf16_hi(v.y);
  f[4] = bf16_lo(v.z); f[5] = bf16_hi(v.z); f[6] = bf16_lo(v.w); f[7] = bf16_hi(v.w);
}

CC_DEV int group_seg(const GemvParams &p, int g) {
  int s = 0;
  while (s + 1 < p.n_seg && g >= p.seg[s + 1].group0) ++s;
  return s;
}

__host__ __device__ inline bool pairs(int epi) { return epi == GEMV_ROPE || epi == GEMV_SWIGLU; }

// First weight row of box `box` (0, 1) of local group gl.  ROPE: the 8
// pairs' first rows, then their partners half a head later; SwiGLU: rows
// gl*8.. of the gate map, then of the up map; otherwise 16 consecutive rows.
CC_DEV int box_row(const GemvParams &p, const GemvSeg &sg, int gl, int box) {
  if (sg.epi == GEMV_ROPE) {
    const int half = p.head_dim >> 1;
    const int u = gl * 8, h = u / half;
    return h * p.head_dim + (u - h * half) + box * half;
  }
  if (sg.epi == GEMV_SWIGLU) return gl * 8;
  return gl * 16 + box * 8;
}

size_t align128(size_t x) { return (x + 127) & ~size_t(127); }

struct SmemLayout {
  size_t xs, res, bars, total;
};

SmemLayout smem_layout(const GemvParams &p) {
  const int piece = kGemvBoxK * p.ks;
  const int kpad = (p.K + piece - 1) / piece * piece;
  SmemLayout L;
  L.xs = (size_t)p.stages * kGemvStageBytes * p.ks;
  L.res = align128(L.xs + (size_t)p.batch * kpad * 2);
  L.bars = align128(L.res + (size_t)2 * kGemvConsumers * p.batch * 4);
  L.total = L.bars + (size_t)(2 * p.stages + 4) * 8;
  return L;
}

template <int KS>
__global__ void __launch_bounds__(kThreads, 1) gemv_kernel(const __grid_constant__ GemvLaunch l,
                                                            unsigned xs_off, unsigned res_off,
                                                            unsigned bars_off) {
  const GemvParams &p = l.p;
  extern __shared__ __align__(1024) uint8_t smem[];
  __shared__ int rows[kGemvMaxRows];
  __shared__ float inv_rms[kGemvMaxRows];
  __shared__ float ssq[kGemvConsumers];
  __shared__ int abort_s;
  volatile int *abort_flag = &abort_s;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  constexpr int kPiece = KS * kGemvBoxK;                // K elements of one stage
  constexpr int kStage = KS * kGemvStageBytes;          // [KS][2 boxes][8 rows][256]
  const int B = p.batch, K = p.K, NS = p.stages;
  const int KC = (K + kPiece - 1) / kPiece, kpad = KC * kPiece;
  uint8_t *ring = smem;
  __nv_bfloat16 *xs = reinterpret_cast<__nv_bfloat16 *>(smem + xs_off);
  float *res = reinterpret_cast<float *>(smem + res_off);
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + bars_off);
  uint64_t *empty = full + NS;
  uint64_t *grp_full = empty + NS;    // [2]: the 16 warps' results of a group are in the slot
  uint64_t *grp_free = grp_full + 2;  // [2]: warp 0 has read the slot
  const int g_begin = (int)((long long)blockIdx.x * p.n_groups / gridDim.x);
  const int g_end = (int)((long long)(blockIdx.x + 1) * p.n_groups / gridDim.x);

  // The next product may launch now: its producer streams its own weights
  // while this grid finishes (every CTA here holds one SM's shared memory,
  // so a waiting dependent never takes an SM this grid still needs).
  pdl_trigger();
  if (threadIdx.x == 0) {
    for (int s = 0; s < NS; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kGemvConsumers);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&grp_full[i], kGemvConsumers);
      mbar_init(&grp_free[i], 1);
    }
    abort_s = 0;
    fence_barrier_init();
  }
  __syncthreads();

  if (warp == kGemvConsumers) {
    // ------------------------------------------------------------ producer
    // (weights only: nothing an earlier kernel writes, so no pdl_wait)
    if (lane == 0) {
      for (int s = 0; s < p.n_seg; ++s) {
        tma_prefetch_desc(&l.w[s][0]);
        if (p.seg[s].epi == GEMV_SWIGLU) tma_prefetch_desc(&l.w[s][1]);
      }
      const uint64_t pol = make_policy_evict_first();
      int s = 0;
      uint32_t ph = 0;
      for (int g = g_begin; g < g_end; ++g) {
        const int si = group_seg(p, g);
        const GemvSeg &sg = p.seg[si];
        const int gl = g - sg.group0;
        const CUtensorMap *m0 = &l.w[si][0];
        const CUtensorMap *m1 = sg.epi == GEMV_SWIGLU ? &l.w[si][1] : m0;
        const int r0 = box_row(p, sg, gl, 0), r1 = box_row(p, sg, gl, 1);
        for (int kc = 0; kc < KC; ++kc) {
          if (!mbar_wait(&empty[s], ph ^ 1u, abort_flag, p.status)) goto producer_done;
          mbar_arrive_expect_tx(&full[s], kStage);
          uint8_t *dst = ring + (size_t)s * kStage;
#pragma unroll
          for (int c = 0; c < KS; ++c) {
            const int k0 = kc * kPiece + c * kGemvBoxK;
            tma_load_2d_hint(dst + c * kGemvStageBytes, m0, &full[s], k0, r0, pol);
            tma_load_2d_hint(dst + c * kGemvStageBytes + kGemvStageBytes / 2, m1, &full[s], k0, r1,
                             pol);
          }
          if (++s == NS) {
            s = 0;
            ph ^= 1u;
          }
        }
      }
    producer_done:;
    }
  } else {
    // ------------------------------------------------------------ consumers
    pdl_wait();   // the rows, the outputs and the row ranges come from earlier kernels
    if (threadIdx.x < B) {
      const int b = threadIdx.x;
      const int lo = p.row_lo[b], hi = p.row_hi[b];
      rows[b] = (hi > lo && lo >= 0 && hi <= p.cap) ? b * p.cap + lo : -1;
    }
    named_barrier_sync(1, kGemvConsumers * 32);
    // 1. stage the batch rows (zeros past K and for rows without a token)
    for (int b = 0; b < B; ++b) {
      const int row = rows[b];
      __nv_bfloat16 *dst = xs + (size_t)b * kpad;
      if (p.norm_gain) {
        const float *xr = reinterpret_cast<const float *>(p.x) + (size_t)max(row, 0) * p.ldx;
        float ss = 0.f;
        if (row >= 0)
          for (int e = threadIdx.x * 4; e < K; e += kGemvConsumers * 32 * 4) {
            const float4 v = *reinterpret_cast<const float4 *>(xr + e);
            ss = fmaf(v.x, v.x, ss);
            ss = fmaf(v.y, v.y, ss);
            ss = fmaf(v.z, v.z, ss);
            ss = fmaf(v.w, v.w, ss);
          }
        ss = warp_sum(ss);
        if (lane == 0) ssq[warp] = ss;
        named_barrier_sync(1, kGemvConsumers * 32);
        if (threadIdx.x == 0) {
          float t = 0.f;
          for (int w = 0; w < kGemvConsumers; ++w) t += ssq[w];
          inv_rms[b] = rsqrtf(t / (float)K + p.eps);
        }
        named_barrier_sync(1, kGemvConsumers * 32);
        const float inv = inv_rms[b];
        for (int e = threadIdx.x * 8; e < kpad; e += kGemvConsumers * 32 * 8) {
          uint4 o = make_uint4(0, 0, 0, 0);
          if (row >= 0 && e < K) {
            const float4 a = *reinterpret_cast<const float4 *>(xr + e);
            const float4 c = *reinterpret_cast<const float4 *>(xr + e + 4);
            float gn[8];
            unpack8f(*reinterpret_cast<const uint4 *>(p.norm_gain + e), gn);
            o.x = pack_bf16x2(a.x * inv * gn[0], a.y * inv * gn[1]);
            o.y = pack_bf16x2(a.z * inv * gn[2], a.w * inv * gn[3]);
            o.z = pack_bf16x2(c.x * inv * gn[4], c.y * inv * gn[5]);
            o.w = pack_bf16x2(c.z * inv * gn[6], c.w * inv * gn[7]);
          }
          *reinterpret_cast<uint4 *>(dst + e) = o;
        }
      } else {
        const __nv_bfloat16 *xr =
            reinterpret_cast<const __nv_bfloat16 *>(p.x) + (size_t)max(row, 0) * p.ldx;
        for (int e = threadIdx.x * 8; e < kpad; e += kGemvConsumers * 32 * 8)
          *reinterpret_cast<uint4 *>(dst + e) = (row >= 0 && e < K)
                                                    ? *reinterpret_cast<const uint4 *>(xr + e)
                                                    : make_uint4(0, 0, 0, 0);
      }
    }
    named_barrier_sync(1, kGemvConsumers * 32);

    // 2. groups
    float am = -INFINITY;   // ARGMAX running (max, first column) of lane b of warp 0
    int ai = -1;
    int s = 0;
    uint32_t ph = 0;
    for (int g = g_begin, gi = 0; g < g_end; ++g, ++gi) {
      float acc[kGemvMaxRows];
#pragma unroll
      for (int b = 0; b < kGemvMaxRows; ++b) acc[b] = 0.f;
      bool ok = true;
      for (int kc = 0; kc < KC; ++kc) {
        if (!(ok = mbar_wait(&full[s], ph, abort_flag, p.status))) break;
        uint4 wv[KS];
#pragma unroll
        for (int c = 0; c < KS; ++c)
          wv[c] = *reinterpret_cast<const uint4 *>(ring + (size_t)s * kStage + c * kGemvStageBytes +
                                                   warp * (kGemvBoxK * 2) + lane * 16);
#pragma unroll
        for (int c = 0; c < KS; ++c) {
          const int k = kc * kPiece + c * kGemvBoxK + lane * 8;
          float wf[8];
          unpack8f(wv[c], wf);
#pragma unroll
          for (int b = 0; b < kGemvMaxRows; ++b) {
            if (b < B) {
              float xf[8];
              unpack8f(*reinterpret_cast<const uint4 *>(xs + (size_t)b * kpad + k), xf);
              float a = acc[b];
#pragma unroll
              for (int e = 0; e < 8; ++e) a = fmaf(wf[e], xf[e], a);
              acc[b] = a;
            }
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[s]);
        if (++s == NS) {
          s = 0;
          ph ^= 1u;
        }
      }
      if (!ok) break;
      const int buf = gi & 1;
      const uint32_t use = (uint32_t)(gi >> 1) & 1u;   // how often this slot was used before, mod 2
      // the slot's previous group (gi - 2) must have been read by warp 0
      if (gi >= 2 && !mbar_wait(&grp_free[buf], use ^ 1u, abort_flag, p.status)) break;
#pragma unroll
      for (int b = 0; b < kGemvMaxRows; ++b) {
        if (b < B) {
          const float v = warp_sum(acc[b]);
          if (lane == 0) res[((size_t)buf * kGemvConsumers + warp) * B + b] = v;
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&grp_full[buf]);
      if (warp != 0) continue;
      // ---- epilogue of group g (warp 0)
      if (!mbar_wait(&grp_full[buf], use, abort_flag, p.status)) break;
      const int si = group_seg(p, g);
      const GemvSeg &sg = p.seg[si];
      const int gl = g - sg.group0;
      const float *rb = res + (size_t)buf * kGemvConsumers * B;
      const int units = pairs(sg.epi) ? 8 : 16;
      if (sg.epi == GEMV_ARGMAX) {
        if (lane < B)
          for (int j = 0; j < units; ++j) {   // columns in increasing order: the first max wins
            const int u = gl * 16 + j;
            const float v = rb[j * B + lane];
            if (u < sg.N && v > am) {
              am = v;
              ai = u;
            }
          }
      } else {
        for (int idx = lane; idx < units * B; idx += 32) {
          const int j = idx / B, b = idx - j * B;
          const int row = rows[b];
          if (row < 0) continue;
          long long orow = row;   // K / V cache row (paged: through the block table)
          if (sg.kv_dest) {
            orow = kv_row(p.pg, p.cap, b, row - b * p.cap);
            if (orow < 0) {
              set_status(p.status, CC_ERR_DEVICE_ARG);
              continue;
            }
          }
          // element index of output column n (head-major cache: head n / head_dim's vector)
          const bool hm = sg.kv_dest && p.pg.head_major;
          auto el = [&](int n) -> size_t {
            if (hm)
              return (((size_t)b * p.pg.hkv + n / p.head_dim) * p.cap + (row - b * p.cap)) *
                         p.head_dim + n % p.head_dim;
            return (size_t)orow * sg.ldo + n;
          };
          if (sg.epi == GEMV_ROPE) {
            const int half = p.head_dim >> 1;
            const int n1 = box_row(p, sg, gl, 0) + j, n2 = n1 + half;
            float a1 = rb[j * B + b], a2 = rb[(8 + j) * B + b];
            if (sg.bias) {
              a1 += __bfloat162float(sg.bias[n1]);
              a2 += __bfloat162float(sg.bias[n2]);
            }
            float c, sn;
            rope_cs((uint32_t)p.pos[row], p.turns[n1 % p.head_dim], c, sn);
            const float y1 = a1 * c - a2 * sn, y2 = a2 * c + a1 * sn;
            if (sg.fp8) {
              uint8_t *o = reinterpret_cast<uint8_t *>(sg.out);
              o[el(n1)] = (uint8_t)pack_e4m3x2(y1 * sg.qscale, 0.f);
              o[el(n2)] = (uint8_t)pack_e4m3x2(y2 * sg.qscale, 0.f);
            } else {
              __nv_bfloat16 *o = reinterpret_cast<__nv_bfloat16 *>(sg.out);
              o[el(n1)] = __float2bfloat16_rn(y1);
              o[el(n2)] = __float2bfloat16_rn(y2);
            }
          } else if (sg.epi == GEMV_SWIGLU) {
            const int u = gl * 8 + j;
            if (u < sg.N)
              reinterpret_cast<__nv_bfloat16 *>(sg.out)[(size_t)row * sg.ldo + u] =
                  __float2bfloat16_rn(silu(rb[j * B + b]) * rb[(8 + j) * B + b]);
          } else {
            const int u = gl * 16 + j;
            if (u >= sg.N) continue;
            const float v = rb[j * B + b];
            if (sg.epi == GEMV_RESID_F32) {
              reinterpret_cast<float *>(sg.out)[(size_t)row * sg.ldo + u] += v;
            } else {
              const float bb = sg.bias ? __bfloat162float(sg.bias[u]) : 0.f;
              if (sg.fp8)
                reinterpret_cast<uint8_t *>(sg.out)[el(u)] =
                    (uint8_t)pack_e4m3x2((v + bb) * sg.qscale, 0.f);
              else
                reinterpret_cast<__nv_bfloat16 *>(sg.out)[el(u)] = __float2bfloat16_rn(v + bb);
            }
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&grp_free[buf]);
    }
    if (warp == 0 && lane < B && p.n_seg == 1 && p.seg[0].epi == GEMV_ARGMAX && rows[lane] >= 0 &&
        !*abort_flag)
      p.part[(size_t)lane * p.part_ld + blockIdx.x] = make_float2(am, __int_as_float(ai));
  }
  __syncthreads();
  if (*abort_flag) __nanosleep(1000000);   // let copies still in flight land
}

}  // namespace

bool gemv_plan(GemvParams &p, int sms) {
  int groups = 0;
  for (int s = 0; s < p.n_seg; ++s) {
    GemvSeg &sg = p.seg[s];
    const int units = sg.epi == GEMV_ROPE ? sg.N / 2 : sg.N;
    const int per = pairs(sg.epi) ? 8 : 16;
    sg.group0 = groups;
    sg.groups = (units + per - 1) / per;
    groups += sg.groups;
  }
  p.n_groups = groups;
  p.ctas = std::min(sms, groups);
  p.part_ld = p.ctas;
  // K chunks per stage: the most (4, 2, 1) that divide K, so no stage holds
  // only fill; the ring holds up to 192 KB
  p.ks = p.K % (4 * kGemvBoxK) == 0 ? 4 : p.K % (2 * kGemvBoxK) == 0 ? 2 : 1;
  p.stages = kGemvMaxStages / p.ks;
  while (p.stages >= 3 && smem_layout(p).total > kGemvSmemMax) --p.stages;
  return p.stages >= 3;
}

size_t gemv_smem_bytes(const GemvParams &p) { return smem_layout(p).total; }

cudaError_t launch_gemv(const GemvLaunch &l, cudaStream_t st) {
  const GemvParams &p = l.p;
  if (p.ctas <= 0) return cudaSuccess;
  if (p.batch < 1 || p.batch > kGemvMaxRows || p.K % 8 || p.ldx % 8 || p.n_seg < 1 ||
      p.n_seg > kGemvMaxSegs || p.stages < 3 || p.stages * p.ks > kGemvMaxStages ||
      (p.ks != 1 && p.ks != 2 && p.ks != 4) ||
      (p.head_dim % 16 && p.seg[0].epi == GEMV_ROPE))
    return cudaErrorInvalidValue;
  const SmemLayout L = smem_layout(p);
  if (L.total > kGemvSmemMax) return cudaErrorInvalidValue;
  static bool attr_set[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 64 && !attr_set[dev]) {
    for (auto kern : {gemv_kernel<1>, gemv_kernel<2>, gemv_kernel<4>}) {
      cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)kGemvSmemMax);
      if (e != cudaSuccess) return e;
    }
    attr_set[dev] = true;
  }
  auto kern = p.ks == 4 ? gemv_kernel<4> : p.ks == 2 ? gemv_kernel<2> : gemv_kernel<1>;
  return launch_pdl(kern, dim3(p.ctas), dim3(kThreads), L.total, st, l, (unsigned)L.xs,
                    (unsigned)L.res, (unsigned)L.bars);
}

}  // namespace cc
