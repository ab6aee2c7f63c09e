// compact.cu -- in-place cache compaction (Algorithm DoMemRefresh:
// K' <- (K' (+) K)_sigma[1:J], V' and X likewise; the kept entries keep
// their relative (time) order).
//
// For every compacted array (K_l, V_l for each layer, H^(L-1), tokens,
// positions) and sequence b: slot k <- slot keep_idx[k], k < keep_count[b].
// keep_idx is strictly ascending, so keep_idx[k] >= k: a destination never
// lies above its source.  Run in parallel, the write of slot k may still
// clobber the source of a LOWER destination k' (keep_idx[k'] = k).
//
// Work units are chunks of consecutive destination slots of one
// (array, sequence), numbered so that chunks of an (array, sequence) come in
// ascending order.  CTAs take unit tickets from an atomic counter (dispatch
// order).  A unit
//   1. reads all its source rows into shared memory (TMA bulk copies for
//      rows of 16-byte multiples; plain loads for 4-byte rows),
//   2. publishes "sources read" for its ticket (release),
//   3. waits (acquire, bounded) until every lower unit of the same
//      (array, sequence) whose source slots overlap its destination slots
//      has published, and
//   4. writes its destination rows.
// A unit only waits on lower tickets, all held by CTAs already running, and
// publishing never waits, so the scheme cannot deadlock.  Each element is
// read once and written once; rows with keep_idx[k] == k (always a prefix)
// are not moved.
#include "compact.cuh"

namespace cc {

namespace {

constexpr int kThreads = 128;

CC_DEV void st_release(unsigned *p, unsigned v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
CC_DEV unsigned ld_acquire(const unsigned *p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Waits until flags[t] != 0; false after kWaitLimitNs (records CC_ERR_TIMEOUT).
CC_DEV bool wait_flag(const unsigned *flag, unsigned *status) {
  if (ld_acquire(flag)) return true;
  const uint64_t t0 = globaltimer();
  for (uint32_t it = 1;; ++it) {
    __nanosleep(64);
    if (ld_acquire(flag)) return true;
    if ((it & 255u) == 0 && globaltimer() - t0 > kWaitLimitNs) {
      set_status(status, CC_ERR_TIMEOUT);
      return false;
    }
  }
}

__global__ void __launch_bounds__(kThreads)
    compact_kernel(const __grid_constant__ CompactParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t *stage = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 127) &
                                               ~uintptr_t(127));
  __shared__ __align__(8) uint64_t bar;
  __shared__ int s_unit, s_go;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (tid == 0) {
    mbar_init(&bar, 1);
    fence_barrier_init();
  }
  if (blockIdx.x == 0) {   // the new lengths; no unit reads seq_len
    for (int b = tid; b < p.batch; b += kThreads) {
      int j = p.keep_count[b];
      p.seq_len[b] = (j >= 0 && j <= p.cap) ? j : 0;
    }
  }
  __syncthreads();
  uint32_t phase = 0;
  volatile int no_abort = 0;

  for (;;) {
    if (tid == 0) s_unit = (int)atomicAdd(p.ticket, 1u);
    __syncthreads();
    const int t = s_unit;
    __syncthreads();
    if (t >= p.total_units) break;
    // ---- locate the unit: array a, sequence b, chunk c
    int a = 0;
    while (a + 1 < p.n_arrays && p.arr[a + 1].unit_base <= t) ++a;
    const CompactArray &A = p.arr[a];
    const int local = t - A.unit_base;
    const int b = local / A.n_chunks, c = local - b * A.n_chunks;
    const int C = A.rows_per_chunk;
    int J = p.keep_count[b];
    if (J < 0 || J > p.cap) {
      if (tid == 0) set_status(p.status, CC_ERR_DEVICE_ARG);
      J = 0;
    }
    const int32_t *kidx = p.keep_idx + (size_t)b * p.cap;
    const int k0 = c * C, k1 = min(k0 + C, J);
    // first moving row: identity rows (kidx[k] == k) form a prefix
    int first = k1;
    if (k0 < k1) {
      if (kidx[k1 - 1] == k1 - 1) {
        first = k1;
      } else if (kidx[k0] != k0) {
        first = k0;
      } else {  // binary search the boundary inside the chunk
        int lo = k0, hi = k1 - 1;   // kidx[lo] == lo, kidx[hi] != hi
        while (hi - lo > 1) {
          int mid = (lo + hi) >> 1;
          if (kidx[mid] == mid) lo = mid; else hi = mid;
        }
        first = hi;
      }
    }
    const size_t seq_off = (size_t)b * p.cap;
    uint8_t *base = reinterpret_cast<uint8_t *>(A.base);
    const int rb = A.row_bytes;
    const bool work = first < k1;

    // ---- 1. read the sources
    if (work) {
      if (A.bulk) {
        if (warp == 0) {
          if (lane == 0) mbar_arrive_expect_tx(&bar, (uint32_t)((k1 - first) * rb));
          __syncwarp();
          for (int k = first + lane; k < k1; k += 32) {
            int src = kidx[k];
            if (src < k || src >= p.cap) {   // not ascending / out of range: copy row onto itself
              set_status(p.status, CC_ERR_DEVICE_ARG);
              src = k;
            }
            bulk_load(stage + (size_t)(k - k0) * rb, base + (seq_off + src) * rb, rb, &bar);
          }
          mbar_wait(&bar, phase, &no_abort, p.status);
        }
        phase ^= 1;
      } else {   // 4-byte rows
        for (int k = first + tid; k < k1; k += kThreads) {
          int src = kidx[k];
          if (src < k || src >= p.cap) {
            set_status(p.status, CC_ERR_DEVICE_ARG);
            src = k;
          }
          reinterpret_cast<uint32_t *>(stage)[k - k0] =
              reinterpret_cast<const uint32_t *>(base)[seq_off + src];
        }
      }
    }
    __syncthreads();
    // ---- 2. publish; 3. wait for lower overlapping units
    if (tid == 0) {
      if (t != p.withhold_unit) st_release(&p.flags[t], 1u);
      int go = 1;
      if (work && c > 0) {
        // highest lower chunk whose first source lies below our last destination
        int lo = 0, hi = c - 1, cand = -1;
        while (lo <= hi) {
          int mid = (lo + hi) >> 1;
          if (kidx[mid * C] < k1) { cand = mid; lo = mid + 1; } else hi = mid - 1;
        }
        for (int c2 = cand; c2 >= 0; --c2) {
          const int last_src = kidx[min((c2 + 1) * C, J) - 1];
          if (last_src < first) break;   // this and all lower chunks read below our rows
          if (!wait_flag(&p.flags[A.unit_base + b * A.n_chunks + c2], p.status)) { go = 0; break; }
        }
      }
      fence_proxy_async_global();
      s_go = go;
    }
    __syncthreads();
    // ---- 4. write the destinations
    if (work && s_go) {
      if (A.bulk) {
        if (warp == 0) {
          fence_proxy_async_global();
          for (int k = first + lane; k < k1; k += 32)
            bulk_store(base + (seq_off + k) * rb, stage + (size_t)(k - k0) * rb, rb);
          bulk_commit();
          bulk_wait_all_read();
        }
      } else {
        for (int k = first + tid; k < k1; k += kThreads)
          reinterpret_cast<uint32_t *>(base)[seq_off + k] =
              reinterpret_cast<const uint32_t *>(stage)[k - k0];
      }
    }
    __syncthreads();
  }
  if (warp == 0) bulk_wait_all();
}

}  // namespace

size_t compact_stage_bytes() { return kStageBytes + 128; }

cudaError_t launch_compact(const CompactParams &p, int grid, cudaStream_t st) {
  static bool attr_set[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 64 && !attr_set[dev]) {
    cudaError_t e = cudaFuncSetAttribute(compact_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)compact_stage_bytes());
    if (e != cudaSuccess) return e;
    attr_set[dev] = true;
  }
  if (p.total_units <= 0) return cudaSuccess;
  compact_kernel<<<grid, kThreads, compact_stage_bytes(), st>>>(p);
  return cudaGetLastError();
}

}  // namespace cc
