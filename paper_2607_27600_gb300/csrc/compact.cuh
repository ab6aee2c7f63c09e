// compact.cuh -- in-place cache compaction kernel.
#pragma once
#include "cc_common.cuh"

namespace cc {

#ifndef CC_COMPACT_STAGE_KB
#define CC_COMPACT_STAGE_KB 12
#endif
#ifndef CC_COMPACT_WARPS
#define CC_COMPACT_WARPS 8
#endif
constexpr int kStageBytes = CC_COMPACT_STAGE_KB * 1024;   // shared-memory staging per unit (two per warp)
constexpr int kMaxCompactArrays = 2 * 128 + 3;
constexpr int kMaxDepClasses = 3;        // distinct chunk sizes (K/V rows, H rows, 4-byte rows)

struct CompactArray {
  void *base;          // [batch][cap][row_bytes]
  int row_bytes;       // bulk arrays: multiple of 16; otherwise 4
  int bulk;            // rows moved by TMA bulk copies
  int rows_per_chunk;  // destination slots per unit
  int n_chunks;        // chunks per sequence = ceil(cap / rows_per_chunk) (upper bound of units)
  int dep_class;       // chunk-size class (index into the readers table)
};

struct CompactParams {
  int batch, cap, n_arrays;
  int total_units;            // upper bound (every chunk of every array and sequence)
  const int32_t *keep_idx;    // [batch][cap]
  const int32_t *keep_count;  // [batch]
  int32_t *seq_len;           // [batch], set to keep_count
  int *unit_base;             // [n_arrays*batch + 1] first unit of each (array, sequence),
                              // written by the planning pre-pass (units past keep_count skipped)
  unsigned *flags;            // [total_units], zeroed before launch
  int2 *deps;                 // readers table, (-1,-1)-filled before launch: per class c,
                              // [batch][class_chunks[c]] at class_offset[c]: first and
                              // last chunk reading sources inside each chunk
  int n_classes;
  int class_rows[kMaxDepClasses];
  int class_chunks[kMaxDepClasses];
  long long class_offset[kMaxDepClasses];
  unsigned *status;
  int withhold_unit;          // test hook: this unit never publishes its flag (-1: none)
  CompactArray arr[kMaxCompactArrays];
};

size_t compact_stage_bytes();
// Launches the pre-passes and the (cooperative) compaction; `sms` = SM count.
cudaError_t launch_compact(const CompactParams &p, int sms, cudaStream_t st);

}  // namespace cc
