// internal.h -- library-internal helpers shared between translation units
// (not part of the C ABI).
#pragma once
#include "compact.cuh"

namespace cc {

// Builds the compaction plan of `cache` (arrays, work units) and the scratch
// bytes it needs; same checks as cc_compact_kv.
cc_status compact_plan_build(const cc_model_cfg *cfg, const cc_kv_cache *cache, CompactParams &p,
                             size_t &scratch_bytes);
// Builds the plan with its scratch at `scratch` and enqueues on `st` the
// clearing of what must start cleared.
cc_status compact_plan_bind(const cc_model_cfg *cfg, const cc_kv_cache *cache, CompactParams &p,
                            void *scratch, cudaStream_t st);
// Status-word address and SM count of the current device.
bool current_device_info(unsigned **status, int *sms);
// Makes `st` wait for the caller's K/V-ready events (cc_kv_cache.kv_ready) of
// layers [l0, l1).
cudaError_t wait_kv_ready(const cc_kv_cache *kv, int l0, int l1, cudaStream_t st);

}  // namespace cc
