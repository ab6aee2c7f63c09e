// cc_common.cuh -- sm_103a building blocks shared by the refresh kernels:
// mbarriers with bounded waits, TMA tensor copies, tcgen05 (UMMA + TMEM)
// wrappers, shared-memory matrix descriptors, the device status word.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

#include "../../include/cc.h"

#define CC_DEV __device__ __forceinline__

namespace cc {

// ---------------------------------------------------------------------------
// device status word (first error wins) and bounded waits
// ---------------------------------------------------------------------------
CC_DEV void set_status(unsigned *status, unsigned code) {
  if (status) atomicCAS(status, 0u, code);
}

CC_DEV uint64_t globaltimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Upper bound of any single wait inside a kernel.  A correct kernel waits
// microseconds; this limit only ends a kernel whose partner never arrives.
constexpr uint64_t kWaitLimitNs = 2000000000ull;

CC_DEV uint32_t smem_u32(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// ---------------------------------------------------------------------------
// mbarrier
// ---------------------------------------------------------------------------
CC_DEV void mbar_init(uint64_t *bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
               : "memory");
}
CC_DEV void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
CC_DEV void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
CC_DEV void mbar_arrive(uint64_t *bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
CC_DEV bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// As mbar_try_wait, with acquire at cluster scope: for a barrier that threads
// of the other CTA of a cluster arrive on (mbar_arrive_cluster).
CC_DEV bool mbar_try_wait_cluster(uint64_t *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Waits for the phase of `parity` to complete.  Gives up (returns false)
// when *abort is set by another role of the CTA, or after kWaitLimitNs, in
// which case it sets *abort and records CC_ERR_TIMEOUT.  CL: acquire at
// cluster scope (arrivals from the other CTA of a pair).
template <bool CL = false>
CC_DEV bool mbar_wait(uint64_t *bar, uint32_t parity, volatile int *abort, unsigned *status) {
  auto try_wait = [&]() { return CL ? mbar_try_wait_cluster(bar, parity) : mbar_try_wait(bar, parity); };
  if (try_wait()) return true;
  uint64_t t0 = globaltimer();
  for (uint32_t it = 1;; ++it) {
    if (try_wait()) return true;
    if ((it & 63u) == 0) {
      if (*abort) return false;
      if (globaltimer() - t0 > kWaitLimitNs) {
        *abort = 1;
        set_status(status, CC_ERR_TIMEOUT);
        return false;
      }
    }
  }
}

// ---------------------------------------------------------------------------
// TMA (cp.async.bulk.tensor) and bulk copies
// ---------------------------------------------------------------------------
CC_DEV void tma_prefetch_desc(const CUtensorMap *m) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(m)) : "memory");
}
CC_DEV void tma_load_2d(void *dst, const CUtensorMap *m, uint64_t *bar, int32_t c0, int32_t c1) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(m)), "r"(smem_u32(bar)), "r"(c0), "r"(c1)
      : "memory");
}
CC_DEV void tma_load_3d(void *dst, const CUtensorMap *m, uint64_t *bar, int32_t c0, int32_t c1,
                        int32_t c2) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(m)), "r"(smem_u32(bar)), "r"(c0), "r"(c1), "r"(c2)
      : "memory");
}
// 2-D tile load with an L2 cache policy (from make_policy_*).
CC_DEV void tma_load_2d_hint(void *dst, const CUtensorMap *m, uint64_t *bar, int32_t c0, int32_t c1,
                             uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%3, %4}], [%2], %5;" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(m)), "r"(smem_u32(bar)), "r"(c0), "r"(c1), "l"(policy)
      : "memory");
}
// 2-D tile load into this CTA's shared memory whose completion is counted
// on the barrier at `bar_cl` (a shared::cluster address): with cta_group::2
// that barrier may belong to the other CTA of the pair, so both CTAs' stage
// loads complete on one barrier of CTA 0.
CC_DEV void tma_load_2d_pair_hint(void *dst, const CUtensorMap *m, uint32_t bar_cl, int32_t c0,
                                  int32_t c1, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      ".L2::cache_hint [%0], [%1, {%3, %4}], [%2], %5;" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(m)), "r"(bar_cl), "r"(c0), "r"(c1), "l"(policy)
      : "memory");
}
// L2 policies: keep (evict last) for data read again soon, stream (evict first).
CC_DEV uint64_t make_policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
CC_DEV uint64_t make_policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
// Barrier among `threads` threads (a multiple of 32) of the CTA, id 1..15.
// Programmatic dependent launch: a kernel launched with the programmatic
// stream-serialization attribute may start before its predecessor in the
// stream has finished.  pdl_trigger: this CTA lets the next such kernel
// launch (it launches once every CTA of this grid has triggered or exited);
// pdl_wait: blocks until the predecessor grid has completed and its writes
// are visible (a no-op for a kernel launched without the attribute).  A
// kernel touches nothing its predecessors write before pdl_wait.
CC_DEV void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
CC_DEV void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

CC_DEV void named_barrier_sync(int id, int threads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}
CC_DEV void st_release_u32(unsigned *p, unsigned v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
CC_DEV unsigned ld_acquire_u32(const unsigned *p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
// Waits until *p == want; false (CC_ERR_TIMEOUT recorded) after kWaitLimitNs.
CC_DEV bool wait_value(const unsigned *p, unsigned want, unsigned *status) {
  if (ld_acquire_u32(p) == want) return true;
  const uint64_t t0 = globaltimer();
  for (uint32_t it = 1;; ++it) {
    __nanosleep(64);
    if (ld_acquire_u32(p) == want) return true;
    if ((it & 255u) == 0 && globaltimer() - t0 > kWaitLimitNs) {
      set_status(status, CC_ERR_TIMEOUT);
      return false;
    }
  }
}
// Contiguous global -> shared copy (16-byte aligned addresses, size % 16 == 0).
CC_DEV void bulk_load(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
          "r"(smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}
// Contiguous shared -> global copy, tracked by bulk async-groups.
CC_DEV void bulk_store(void *dst, const void *src, uint32_t bytes) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst),
               "r"(smem_u32(src)), "r"(bytes)
               : "memory");
}
CC_DEV void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
CC_DEV void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
CC_DEV void bulk_wait_all_read() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
CC_DEV void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
CC_DEV void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

// ---------------------------------------------------------------------------
// tcgen05: tensor memory and the 5th-generation MMA
// ---------------------------------------------------------------------------
// Allocation is warp-wide; writes the TMEM base address to *dst (shared).
CC_DEV void tmem_alloc(uint32_t *dst, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(dst)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
CC_DEV void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
CC_DEV void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
CC_DEV void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// D[tmem] (+)= A[smem desc] * B[smem desc]^T, kind::f16 (bf16 in, fp32 acc).
CC_DEV void umma_ss(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                    uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// D[tmem] (+)= A[tmem] * B[smem desc]^T.
CC_DEV void umma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                    uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive on `bar` once every tcgen05 op this thread issued so far completes.
CC_DEV void umma_commit(uint64_t *bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}

// ---------------------------------------------------------------------------
// CTA pairs: a cluster of two CTAs on two SMs sharing one tcgen05 product
// (cta_group::2).  The pair's M = 256 product reads A rows 0-127 from the
// shared memory of CTA 0 and rows 128-255 from CTA 1, B rows [0, N/2) from
// CTA 0 and [N/2, N) from CTA 1 (both at the same shared-memory offsets), and
// writes D rows 0-127 to the tensor memory of CTA 0 and 128-255 to CTA 1.
// One thread of CTA 0 issues it; allocation and release of the tensor
// memory are done by one warp of each CTA together.
// ---------------------------------------------------------------------------
CC_DEV uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
CC_DEV uint32_t cluster_nctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
  return r;
}
// Address in the shared::cluster window of the variable at `p` (this CTA's
// shared memory) as laid out in CTA `rank` of the cluster.
CC_DEV uint32_t cluster_addr(const void *p, uint32_t rank) {
  uint32_t a;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(a) : "r"(smem_u32(p)), "r"(rank));
  return a;
}
// Arrive on an mbarrier of another CTA of the cluster (release, cluster scope).
CC_DEV void mbar_arrive_cluster(uint32_t cl_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cl_addr)
               : "memory");
}
// Every thread of every CTA of the cluster (release / acquire).
CC_DEV void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\t"
               "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
CC_DEV void tmem_alloc_pair(uint32_t *dst, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(dst)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
CC_DEV void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
// The pair's D[tmem] (+)= A[smem desc] * B[smem desc]^T (kind::f16), issued
// by CTA 0 for both CTAs.
CC_DEV void umma_ss_pair(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                         uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive on the mbarrier at `bar`'s offset in every CTA of `cta_mask` once
// the pair products this thread issued so far complete.
CC_DEV void umma_commit_pair(uint64_t *bar, uint16_t cta_mask) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(smem_u32(bar)),
      "h"(cta_mask)
      : "memory");
}

// Instruction descriptor for kind::f16: bf16 A and B, fp32 D, M x N tile.
// a_mn / b_mn: operand stored MN-major (1) rather than K-major (0).
__host__ __device__ constexpr uint32_t make_idesc_bf16(int M, int N, int a_mn, int b_mn) {
  return (1u << 4)                          // D format: f32
         | (1u << 7)                        // A format: bf16
         | (1u << 10)                       // B format: bf16
         | (uint32_t(a_mn) << 15) | (uint32_t(b_mn) << 16)
         | (uint32_t(N >> 3) << 17)         // N / 8
         | (uint32_t(M >> 4) << 24);        // M / 16
}

// Instruction descriptor for kind::f16 with f16 A and B (A and B always share
// one type), fp32 D.
__host__ __device__ constexpr uint32_t make_idesc_f16(int M, int N, int a_mn, int b_mn) {
  return (1u << 4)                          // D format: f32
         | (0u << 7)                        // A format: f16
         | (0u << 10)                       // B format: f16
         | (uint32_t(a_mn) << 15) | (uint32_t(b_mn) << 16)
         | (uint32_t(N >> 3) << 17)         // N / 8
         | (uint32_t(M >> 4) << 24);        // M / 16
}

// Shared-memory matrix descriptor, 128-byte swizzle (rows of 128 bytes,
// 8-row / 1024-byte swizzle atoms).  lbo/sbo in bytes.
CC_DEV uint64_t make_sdesc_sw128(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  return uint64_t((saddr & 0x3FFFFu) >> 4) | (uint64_t((lbo >> 4) & 0x3FFFu) << 16) |
         (uint64_t((sbo >> 4) & 0x3FFFu) << 32) | (1ull << 46) | (2ull << 61);
}

// 32 lanes x 32 consecutive 32-bit columns (one row per thread).
CC_DEV void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
      "%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}
CC_DEV void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

CC_DEV void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,"
      "%13,%14,%15,%16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
      "r"(r[15])
      : "memory");
}
CC_DEV void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,"
      "%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(
          taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
      "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]),
      "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]),
      "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}
CC_DEV void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// Launches kern<<<grid, block, smem, st>>>(args...) with programmatic stream
// serialization allowed (see pdl_wait).
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t st, Args &&...args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

// ---------------------------------------------------------------------------
// small numeric helpers
// ---------------------------------------------------------------------------
CC_DEV uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t *>(&v);
}
CC_DEV float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
CC_DEV float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xFFFF0000u); }
CC_DEV uint32_t pack_f16x2(float lo, float hi) {
  __half2 v = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<uint32_t *>(&v);
}

// Largest finite fp16 value.  The fp16 operand mode (CC_SCORE_F16) reports
// a value written as an fp16 operand whose magnitude exceeds it.
constexpr float kF16Max = 65504.f;

// A finite value that fp16 cannot hold (its magnitude above kF16Max).
CC_DEV bool f16_overflow(float x) {
  const float a = fabsf(x);
  return a > kF16Max && a < INFINITY;
}

// Two activations as the next tensor-core product reads them: a bf16 pair,
// or an fp16 pair (f16), recording in `over` a finite magnitude above
// kF16Max (infinities and NaN pass through unflagged).
CC_DEV uint32_t pack_act2(float lo, float hi, bool f16, bool &over) {
  if (f16) {
    over |= f16_overflow(lo) || f16_overflow(hi);
    return pack_f16x2(lo, hi);
  }
  return pack_bf16x2(lo, hi);
}

// K/V layout.  Paged K/V: the pool row of logical slot i of sequence b.  Pages hold `page`
// slots (a multiple of 128, so a key tile never straddles two pages); the
// block table has pages_per_seq entries per sequence.  Without a table the
// buffers are slot-major: row b * cap + i.  An entry outside [0, n_pages)
// gives -1 (callers skip the row and report it).
// Head-major buffers ([batch][Hkv][cap][head_dim], not paged) keep each KV
// head's vectors of a sequence contiguous instead.
struct KvLayout {
  const int32_t *table;   // device [batch][pages_per_seq], or nullptr
  int page, pages_per_seq, n_pages;
  int head_major;         // [batch][Hkv][cap][head_dim]
  int hkv;                // KV heads
};
CC_DEV long long kv_row(const KvLayout &pg, int cap, int b, int i) {
  if (!pg.table) return (long long)b * cap + i;
  const int e = pg.table[(size_t)b * pg.pages_per_seq + i / pg.page];
  if (e < 0 || e >= pg.n_pages) return -1;
  return (long long)e * pg.page + i % pg.page;
}
// Index (in head_dim-element vectors) of KV head g's vector of slot i of
// sequence b in the K or V buffer; -1 for a bad page.
CC_DEV long long kv_vec(const KvLayout &L, int cap, int b, int g, int i) {
  if (L.head_major) return ((long long)b * L.hkv + g) * cap + i;
  const long long r = kv_row(L, cap, b, i);
  return r < 0 ? -1 : r * L.hkv + g;
}

// Two e4m3 codes (lo in the low byte): round to nearest even, saturating to
// +-448 (the e4m3 K/V cache's element encoding).
CC_DEV uint32_t pack_e4m3x2(float lo, float hi) {
  unsigned short r;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(r) : "f"(hi), "f"(lo));
  return r;
}

CC_DEV float silu(float x) { return x / (1.0f + __expf(-x)); }

// cos/sin of pos * inv_freq, with the angle reduced exactly: turns is
// inv_freq / (2 pi) in 0.64 fixed point, so pos * turns mod 2^64 is the
// fractional number of turns; its top 32 bits, read as a signed fraction of
// a turn, give the angle in [-pi, pi).
CC_DEV void rope_cs(uint32_t pos, unsigned long long turns, float &c, float &s) {
  unsigned long long frac = (unsigned long long)pos * turns;
  int32_t t32 = (int32_t)(frac >> 32);
  float ang = (float)t32 * 1.4629180792671596e-09f;   // 2 pi / 2^32
  __sincosf(ang, &s, &c);
}

CC_DEV float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
  return v;
}
CC_DEV float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
  return v;
}

// Row tiles of a ragged batch: sequence b contributes the rows (slots)
// [row_lo[b], seq_len[b]) in ceil((seq_len[b] - row_lo[b]) / tile) tiles of
// `tile` rows.  prefix[b] = first tile of sequence b (prefix[batch] = total).
// Invalid ranges (outside [0, cap]) count as 0 and are reported.
// seq_len == nullptr means every sequence ends at cap; row_lo == nullptr
// means every range starts at slot 0.
CC_DEV int build_tile_prefix(const int32_t *seq_len, const int32_t *row_lo, int batch, int cap,
                             int tile, int *prefix, unsigned *status) {
  int acc = 0;
  for (int b = 0; b < batch; ++b) {
    prefix[b] = acc;
    const int hi = seq_len ? seq_len[b] : cap;
    const int lo = row_lo ? row_lo[b] : 0;
    int n = hi - lo;
    if (lo < 0 || hi > cap || n < 0) {
      set_status(status, CC_ERR_DEVICE_ARG);
      n = 0;
    }
    acc += (n + tile - 1) / tile;
  }
  prefix[batch] = acc;
  return acc;
}
CC_DEV int find_seq(const int *prefix, int batch, int t) {
  int lo = 0, hi = batch - 1;
  while (lo < hi) {  // last b with prefix[b] <= t
    int mid = (lo + hi + 1) >> 1;
    if (prefix[mid] <= t) lo = mid; else hi = mid - 1;
  }
  return lo;
}

}  // namespace cc
