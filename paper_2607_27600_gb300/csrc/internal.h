// internal.h -- library-internal helpers shared between translation units
// (not part of the C ABI).
#pragma once
#include "compact.cuh"

namespace cc {

// Builds the compaction plan of `cache` (arrays, work units; the same checks
// as cc_compact_kv) once, rejects it with CC_ERR_WORKSPACE when its scratch
// exceeds `scratch_cap` bytes, else places the scratch at `scratch` and
// enqueues on `st` the clearing of what must start cleared.
cc_status compact_plan_bind(const cc_model_cfg *cfg, const cc_kv_cache *cache, CompactParams &p,
                            void *scratch, size_t scratch_cap, cudaStream_t st);
// launch_compact inside the same launch-timing scope as cc_compact_kv's
// (cc_profile.h, kind CC_KERNEL_COMPACT).
cudaError_t launch_compact_timed(const CompactParams &p, int sms, cudaStream_t st);
// Status-word address and SM count of the current device.
bool current_device_info(unsigned **status, int *sms);
// Makes `st` wait for the caller's K/V-ready events (cc_kv_cache.kv_ready) of
// layers [l0, l1).
cudaError_t wait_kv_ready(const cc_kv_cache *kv, int l0, int l1, cudaStream_t st);

}  // namespace cc
