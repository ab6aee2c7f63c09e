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
// (array, sequence), numbered so that the chunks of an (array, sequence)
// come in ascending order.  A unit
//   1. reads all its source rows into shared memory (TMA bulk copies for
//      rows of 16-byte multiples; plain loads for 4-byte rows),
//   2. publishes "sources read" for its unit (release),
//   3. waits (acquire, bounded) until every lower unit that reads from its
//      destination slots has published, and
//   4. writes its destination rows (bulk stores).
// Which lower units read from a chunk is found once per refresh by a small
// pre-pass over keep_idx (deps_kernel): chunk u's readers are the chunks
// holding the first and last k with keep_idx[k] in u.
//
// A planning pre-pass numbers only the units that hold kept slots.  The
// kernel is launched cooperatively (every warp resident) and warp w takes
// units w, w + W, w + 2W, ... in ascending order, no atomics.  A unit waits
// only on lower units and publishing never waits: the lowest unpublished
// unit's warp is never blocked, so nothing can deadlock.  Each warp runs its
// own two-buffer pipeline: the loads of its next unit are in flight while
// the current unit waits and stores.  Each element is read once and written
// once; rows with keep_idx[k] == k are not moved.
#include "compact.cuh"

namespace cc {

namespace {

constexpr int kThreads = kCompactMaxWarps * 32;   // launch bound; p.warps warps run

CC_DEV void st_release(unsigned *p, unsigned v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
CC_DEV unsigned ld_acquire(const unsigned *p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Waits until *flag != 0; false after kWaitLimitNs (records CC_ERR_TIMEOUT).
CC_DEV bool wait_flag(const unsigned *flag, unsigned *status) {
  if (ld_acquire(flag)) return true;
  const uint64_t t0 = globaltimer();
  for (uint32_t it = 1;; ++it) {
    __nanosleep(32);
    if (ld_acquire(flag)) return true;
    if ((it & 255u) == 0 && globaltimer() - t0 > kWaitLimitNs) {
      set_status(status, CC_ERR_TIMEOUT);
      return false;
    }
  }
}

// Pre-pass: for every chunk u of class cls (chunks of class_rows[cls] slots),
// the first and last chunk whose destinations read sources inside u.
__global__ void deps_kernel(const __grid_constant__ CompactParams p) {
  const int cls = blockIdx.z, b = blockIdx.y;
  const int k = blockIdx.x * blockDim.x + threadIdx.x;
  int J = p.keep_count[b];
  if (J < 0 || J > p.cap) J = 0;
  if (k >= J) return;
  const int C = p.class_rows[cls];
  const int32_t *kidx = p.keep_idx + (size_t)b * p.cap;
  auto src_of = [&](int kk) {
    int s = kidx[kk];
    return (s < kk || s >= p.cap) ? kk : s;   // invalid entries are copied onto themselves
  };
  const int u = src_of(k) / C;
  int2 *deps = p.deps + p.class_offset[cls] + (size_t)b * p.class_chunks[cls];
  if (k == 0 || src_of(k - 1) / C != u) deps[u].x = k / C;
  if (k == J - 1 || src_of(k + 1) / C != u) deps[u].y = k / C;
}

// Pre-pass: unit_base[a*batch + b] = first unit of (array a, sequence b),
// counting ceil(keep_count[b] / rows_per_chunk) units each; the last entry
// is the number of units.  One block: an exclusive scan over the
// (array, sequence) pairs, 1024 pairs per round.
__global__ void __launch_bounds__(1024) plan_kernel(const __grid_constant__ CompactParams p) {
  __shared__ int warp_sums[32];
  __shared__ int carry;
  const int n_pairs = p.n_arrays * p.batch;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) carry = 0;
  __syncthreads();
  for (int base = 0; base < n_pairs; base += 1024) {
    const int t = base + threadIdx.x;
    int units = 0;
    if (t < n_pairs) {
      const int a = t / p.batch, b = t - a * p.batch;
      const int C = p.arr[a].rows_per_chunk;
      int J = p.keep_count[b];
      if (J < 0 || J > p.cap) {
        if (a == 0) set_status(p.status, CC_ERR_DEVICE_ARG);
        J = 0;
      }
      units = (J + C - 1) / C;
    }
    int incl = units;   // inclusive scan within the warp
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xFFFFFFFFu, incl, o);
      if (lane >= o) incl += v;
    }
    if (lane == 31) warp_sums[warp] = incl;
    __syncthreads();
    if (warp == 0) {
      const int ws = warp_sums[lane];
      int wi = ws;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int v = __shfl_up_sync(0xFFFFFFFFu, wi, o);
        if (lane >= o) wi += v;
      }
      warp_sums[lane] = wi - ws;   // exclusive prefix of the warp totals
    }
    __syncthreads();
    const int excl = carry + warp_sums[warp] + incl - units;
    if (t < n_pairs) p.unit_base[t] = excl;
    __syncthreads();
    if (threadIdx.x == 1023) carry = excl + units;
    __syncthreads();
  }
  if (threadIdx.x == 0) p.unit_base[n_pairs] = carry;
}

struct Unit {
  int t;          // unit number (>= total: none)
  int a, b, c;    // array, sequence, chunk
  int k0, k1;     // destination slots [k0, k1)
  bool loaded;    // bulk loads issued into the buffer
};

__global__ void __launch_bounds__(kThreads)
    compact_kernel(const __grid_constant__ CompactParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 127) &
                                              ~uintptr_t(127));
  __shared__ __align__(8) uint64_t bars[kCompactMaxWarps][2];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int n_warps = p.warps;
  uint8_t *buf[2] = {smem + (size_t)(warp * 2 + 0) * p.stage_bytes,
                     smem + (size_t)(warp * 2 + 1) * p.stage_bytes};
  if (lane == 0) {
    mbar_init(&bars[warp][0], 1);
    mbar_init(&bars[warp][1], 1);
    fence_barrier_init();
  }
  if (blockIdx.x == 0 && warp == 0) {   // the new lengths; no unit reads seq_len
    for (int b = lane; b < p.batch; b += 32) {
      int j = p.keep_count[b];
      p.seq_len[b] = (j >= 0 && j <= p.cap) ? j : 0;
    }
  }
  const int n_pairs = p.n_arrays * p.batch;
  int *ub_smem = reinterpret_cast<int *>(smem + (size_t)n_warps * 2 * p.stage_bytes);
  if (p.ub_cached)
    for (int i = threadIdx.x; i <= n_pairs; i += blockDim.x) ub_smem[i] = p.unit_base[i];
  __syncthreads();
  const int *unit_base = p.ub_cached ? ub_smem : p.unit_base;
  uint32_t phase[2] = {0, 0};
  volatile int no_abort = 0;

  const int total = unit_base[n_pairs];
  const int stride = gridDim.x * n_warps;
  int next_t = blockIdx.x * n_warps + warp;
  auto take = [&]() -> Unit {
    Unit u;
    u.t = next_t;
    next_t += stride;
    u.loaded = false;
    u.a = u.b = u.c = u.k0 = u.k1 = 0;
    if (u.t >= total) return u;
    int lo = 0, hi = n_pairs - 1;   // last pair whose first unit <= t
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (unit_base[mid] <= u.t) lo = mid; else hi = mid - 1;
    }
    u.a = lo / p.batch;
    u.b = lo - u.a * p.batch;
    u.c = u.t - unit_base[lo];
    const CompactArray &A = p.arr[u.a];
    int J = p.keep_count[u.b];
    if (J < 0 || J > p.cap) J = 0;
    u.k0 = u.c * A.rows_per_chunk;
    u.k1 = min(u.k0 + A.rows_per_chunk, J);
    return u;
  };

  // Source row of destination k; entries that are not ascending or out of
  // range are copied onto themselves (and reported by `report`).
  auto source = [&](const int32_t *kidx, int k, bool report) {
    int s = kidx[k];
    if (s < k || s >= p.cap) {
      if (report) set_status(p.status, CC_ERR_DEVICE_ARG);
      s = k;
    }
    return s;
  };

  // Row of slot k of sequence b in array A (paged K/V: the pool row, -1 for
  // a bad block-table entry, which is reported and its row left alone).
  auto arow = [&](const CompactArray &A, int b, int k) -> long long {
    if (!A.paged) return (long long)b * p.cap + k;
    const long long r = kv_row(p.pg, p.cap, b, k);
    if (r < 0) set_status(p.status, CC_ERR_DEVICE_ARG);
    return r;
  };
  // Copies one bulk row (slot k of sequence b) between global memory and a
  // shared-memory row; head-major arrays move it as Hkv segments.
  auto row_load = [&](const CompactArray &A, int b, int src, uint8_t *dst, uint64_t *bar) {
    uint8_t *base = reinterpret_cast<uint8_t *>(A.base);
    if (A.head_major) {
      const int seg = A.row_bytes / p.pg.hkv;
      for (int g = 0; g < p.pg.hkv; ++g)
        bulk_load(dst + g * seg, base + (((size_t)b * p.pg.hkv + g) * p.cap + src) * seg, seg, bar);
    } else {
      bulk_load(dst, base + (size_t)arow(A, b, src) * A.row_bytes, A.row_bytes, bar);
    }
  };
  auto row_store = [&](const CompactArray &A, int b, int k, const uint8_t *src) {
    uint8_t *base = reinterpret_cast<uint8_t *>(A.base);
    if (A.head_major) {
      const int seg = A.row_bytes / p.pg.hkv;
      for (int g = 0; g < p.pg.hkv; ++g)
        bulk_store(base + (((size_t)b * p.pg.hkv + g) * p.cap + k) * seg, src + g * seg, seg);
    } else {
      bulk_store(base + (size_t)arow(A, b, k) * A.row_bytes, src, A.row_bytes);
    }
  };
  // A bulk row moves when its source differs and both rows exist.
  auto moves = [&](const CompactArray &A, int b, int k, int src) {
    return src != k && (!A.paged || (arow(A, b, k) >= 0 && arow(A, b, src) >= 0));
  };

  // Issues the reads of unit u into buffer slot s.
  auto load = [&](Unit &u, int s) {
    if (u.t >= total || u.k0 >= u.k1) return;
    const CompactArray &A = p.arr[u.a];
    const int32_t *kidx = p.keep_idx + (size_t)u.b * p.cap;
    uint8_t *base = reinterpret_cast<uint8_t *>(A.base);
    const size_t seq_off = (size_t)u.b * p.cap;
    if (A.bulk) {
      int moving = 0;
      for (int k = u.k0 + lane; k < u.k1; k += 32) moving += moves(A, u.b, k, source(kidx, k, false));
      moving = __reduce_add_sync(0xFFFFFFFFu, moving);
      if (moving == 0) return;
      if (lane == 0) mbar_arrive_expect_tx(&bars[warp][s], (uint32_t)(moving * A.row_bytes));
      __syncwarp();
      for (int k = u.k0 + lane; k < u.k1; k += 32) {
        const int src = source(kidx, k, true);
        if (moves(A, u.b, k, src))
          row_load(A, u.b, src, buf[s] + (size_t)(k - u.k0) * A.row_bytes, &bars[warp][s]);
      }
      u.loaded = true;
    } else {   // 4-byte rows: plain loads staged in shared memory
      uint32_t *st = reinterpret_cast<uint32_t *>(buf[s]);
#pragma unroll 8
      for (int k = u.k0 + lane; k < u.k1; k += 32)
        st[k - u.k0] = reinterpret_cast<const uint32_t *>(base)[seq_off + source(kidx, k, true)];
    }
  };

  Unit cur = take();
  load(cur, 0);
  Unit nxt = take();
  load(nxt, 1);
  for (int i = 0; cur.t < total; ++i) {
    const int s = i & 1;
    const CompactArray &A = p.arr[cur.a];
    // ---- 1. sources of `cur` are in shared memory
    if (cur.loaded) {
      mbar_wait(&bars[warp][s], phase[s], &no_abort, p.status);
      phase[s] ^= 1;
    }
    __syncwarp();
    // ---- 2. publish; 3. wait for the lower units that read our destinations
    // A unit is waited on exactly when one of its source chunks is an active
    // destination chunk above its own (the readers table lists it there), so
    // only such units publish (a release store costs a memory barrier).
    bool go = true;
    if (lane == 0) {
      if (cur.k0 < cur.k1) {
        const int32_t *kidx = p.keep_idx + (size_t)cur.b * p.cap;
        const int C = A.rows_per_chunk;
        int J = p.keep_count[cur.b];
        J = (J < 0 || J > p.cap) ? 0 : J;
        const int active = (J + C - 1) / C;
        const int lo_u = max(cur.c + 1, source(kidx, cur.k0, false) / C);
        const int hi_u = min(active - 1, source(kidx, cur.k1 - 1, false) / C);
        if (lo_u <= hi_u && cur.t != p.withhold_unit) st_release(&p.flags[cur.t], 1u);
      }
      bool waited = false;
      if (cur.k0 < cur.k1 && cur.c > 0) {
        const int2 d = p.deps[p.class_offset[A.dep_class] +
                              (size_t)cur.b * p.class_chunks[A.dep_class] + cur.c];
        const int hi = min(d.y, cur.c - 1);
        for (int c2 = max(d.x, 0); c2 <= hi && go; ++c2) {
          go = wait_flag(&p.flags[unit_base[cur.a * p.batch + cur.b] + c2], p.status);
          waited = true;
        }
      }
      if (waited) fence_proxy_async_global();
    }
    go = __shfl_sync(0xFFFFFFFFu, go ? 1 : 0, 0) != 0;
    // ---- 4. write the destinations
    if (go && cur.k0 < cur.k1) {
      const int32_t *kidx = p.keep_idx + (size_t)cur.b * p.cap;
      uint8_t *base = reinterpret_cast<uint8_t *>(A.base);
      const size_t seq_off = (size_t)cur.b * p.cap;
      if (A.bulk) {
        if (cur.loaded) {
          for (int k = cur.k0 + lane; k < cur.k1; k += 32)
            if (moves(A, cur.b, k, source(kidx, k, false)))
              row_store(A, cur.b, k, buf[s] + (size_t)(k - cur.k0) * A.row_bytes);
          bulk_commit();
        }
      } else {
        const uint32_t *st = reinterpret_cast<const uint32_t *>(buf[s]);
        for (int k = cur.k0 + lane; k < cur.k1; k += 32)
          reinterpret_cast<uint32_t *>(base)[seq_off + k] = st[k - cur.k0];
      }
    }
    bulk_wait_all_read();   // buffer s may be refilled
    __syncwarp();
    Unit nn = take();
    load(nn, s);
    cur = nxt;
    nxt = nn;
  }
  bulk_wait_all();
}

}  // namespace

bool compact_shape(int max_row_bytes, int &stage_bytes, int &warps) {
  stage_bytes = kCompactStageBytes;
  if (max_row_bytes > stage_bytes) stage_bytes = (max_row_bytes + 127) & ~127;
  warps = kCompactTargetBytes / (2 * stage_bytes);
  if (warps > kCompactMaxWarps) warps = kCompactMaxWarps;
  if (warps < 1 && 2 * stage_bytes + 128 <= kCompactSmemBytes) warps = 1;
  return warps >= 1;
}

void compact_cache_units(CompactParams &p) {
  const size_t table = (((size_t)p.n_arrays * p.batch + 1) * sizeof(int) + 15) & ~size_t(15);
  p.ub_cached = (size_t)p.warps * 2 * p.stage_bytes + 128 + table <= (size_t)kCompactSmemBytes;
}

size_t compact_smem_bytes(const CompactParams &p) {
  const size_t table = p.ub_cached ? ((size_t)p.n_arrays * p.batch + 1) * sizeof(int) : 0;
  return (size_t)p.warps * 2 * p.stage_bytes + 128 + ((table + 15) & ~size_t(15));
}

cudaError_t launch_compact(const CompactParams &p, int sms, cudaStream_t st) {
  // resident CTAs per SM for this shape (the cooperative launch needs all of them)
  static bool attr_set[64] = {};
  static int occ_cache[64][kCompactMaxWarps + 1] = {};
  static int occ_smem[64][kCompactMaxWarps + 1] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (p.warps < 1 || p.warps > kCompactMaxWarps || p.stage_bytes < 16) return cudaErrorInvalidValue;
  const size_t smem = compact_smem_bytes(p);
  if (!attr_set[dev]) {
    cudaError_t e = cudaFuncSetAttribute(compact_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kCompactSmemBytes);
    if (e != cudaSuccess) return e;
    attr_set[dev] = true;
  }
  if (occ_smem[dev][p.warps] != (int)smem) {
    int n = 0;
    cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, compact_kernel, p.warps * 32,
                                                                  smem);
    if (e != cudaSuccess) return e;
    if (n < 1) return cudaErrorLaunchOutOfResources;
    occ_cache[dev][p.warps] = n;
    occ_smem[dev][p.warps] = (int)smem;
  }
  const int blocks_per_sm = occ_cache[dev][p.warps];
  if (p.total_units <= 0) return cudaSuccess;
  for (int cls = 0; cls < p.n_classes; ++cls) {
    if (p.class_rows[cls] <= 0) return cudaErrorInvalidValue;
  }
  plan_kernel<<<1, 1024, 0, st>>>(p);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const dim3 dgrid((p.cap + 255) / 256, p.batch, p.n_classes);
  deps_kernel<<<dgrid, 256, 0, st>>>(p);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  // cooperative: every warp resident, so the static unit order cannot deadlock
  void *args[] = {const_cast<CompactParams *>(&p)};
  return cudaLaunchCooperativeKernel((const void *)compact_kernel, dim3(sms * blocks_per_sm),
                                     dim3(p.warps * 32), args, smem, st);
}

}  // namespace cc
