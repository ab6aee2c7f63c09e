// internal.h -- library-internal helpers shared between translation units
// (not part of the C ABI).
#pragma once
#include "compact.cuh"

namespace cc {

// Builds the compaction plan of `cache` (arrays, work units) and the scratch
// bytes it needs (the first flags_bytes start at zero, the rest at 0xFF);
// same checks as cc_compact_kv.
cc_status compact_plan_build(const cc_model_cfg *cfg, const cc_kv_cache *cache, CompactParams &p,
                             size_t &flags_bytes, size_t &scratch_bytes);
// Status-word address and SM count of the current device.
bool current_device_info(unsigned **status, int *sms);

}  // namespace cc
