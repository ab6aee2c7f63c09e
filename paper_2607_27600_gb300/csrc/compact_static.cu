// compact_static.cu -- cc_compact_kv_static: the in-place compaction of
// cc_compact_kv for callers that cannot allocate device memory.
//
// cc_compact_kv takes its scratch (a table of work units, one "sources read"
// flag per unit and a table of which units read each destination chunk) from
// a caller-provided workspace.  This
// variant takes it from a fixed array in the library's own device memory
// instead, so the caller passes only the cache, the keep-set and a stream.
// The array is a file-scope __device__ variable: every GPU that loads the
// library holds its kStaticScratchBytes until the process exits, and every
// call on a device shares it.
#include <mutex>

#include "internal.h"

namespace {

// 1 MiB: the unit table (4 bytes per array and sequence), one 4-byte flag
// per work unit and the readers table (8 bytes per destination chunk).
constexpr size_t kStaticScratchBytes = size_t(1) << 20;
__device__ __align__(256) unsigned char g_compact_scratch[kStaticScratchBytes];

constexpr int kMaxDevices = 64;
// Device address of g_compact_scratch per device.  In host code the symbol
// name is only a host-side stand-in, never a device address.
unsigned char *g_scratch_addr[kMaxDevices] = {};
std::mutex g_scratch_mu;

cc_status scratch_address(unsigned char **out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return CC_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_scratch_mu);
  if (!g_scratch_addr[dev]) {   // set-up, once per device, with that device current
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_compact_scratch) != cudaSuccess || !p) return CC_ERR_CUDA;
    g_scratch_addr[dev] = static_cast<unsigned char *>(p);
  }
  *out = g_scratch_addr[dev];
  return CC_OK;
}

}  // namespace

extern "C" cc_status cc_compact_kv_static(const cc_model_cfg *cfg, const cc_kv_cache *cache,
                                          const int32_t *keep_idx, const int32_t *keep_count,
                                          void *stream) {
  static cc::CompactParams p;   // large kernel-parameter block; guarded by mu
  static std::mutex mu;
  std::lock_guard<std::mutex> lk(mu);
  if (!cfg || !cache) return CC_ERR_INVALID_ARG;
  if (!keep_idx || !keep_count) return CC_ERR_INVALID_ARG;
  unsigned char *scratch = nullptr;
  cc_status s = scratch_address(&scratch);
  if (s != CC_OK) return s;
  unsigned *status = nullptr;
  int sms = 0;
  if (!cc::current_device_info(&status, &sms)) return CC_ERR_CUDA;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  // one plan build: rejected (CC_ERR_WORKSPACE, nothing enqueued) when its
  // scratch exceeds the array; else the flags start at zero and the readers
  // table at -1 (cleared on `st`), since the array keeps the last call's contents
  if ((s = cc::compact_plan_bind(cfg, cache, p, scratch, kStaticScratchBytes, st)) != CC_OK)
    return s;
  p.keep_idx = keep_idx;
  p.keep_count = keep_count;
  p.seq_len = cache->seq_len;
  p.status = status;
  if (cc::wait_kv_ready(cache, 0, cfg->n_layers, st) != cudaSuccess) return CC_ERR_CUDA;
  if (cc::launch_compact_timed(p, sms, st) != cudaSuccess) return CC_ERR_CUDA;
  return CC_OK;
}
