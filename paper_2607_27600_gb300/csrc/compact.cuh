// compact.cuh -- in-place cache compaction kernel.
#pragma once
#include "cc_common.cuh"

namespace cc {

// Each warp of the copy kernel runs a two-buffer pipeline of units; a unit
// stages up to one buffer of rows in shared memory.  The buffer is 4 KB, or
// the largest row the cache moves if that is larger, and a CTA runs as many
// warps as fill ~192 KB of staging (at most 24): measured fastest on
// Llama-3-8B caches, 24 x 2 x 4 KB when only 2 KB K/V rows move, 12 x 2 x
// 8 KB with 8 KB H^(L-1) rows.  Rows up to ~112 KB are supported (one warp).
constexpr int kCompactMaxWarps = 24;
constexpr int kCompactStageBytes = 4 * 1024;
constexpr int kCompactTargetBytes = 192 * 1024;   // staging the shape aims for
constexpr int kCompactSmemBytes = 224 * 1024;     // dynamic shared memory limit of the copy kernel
constexpr int kMaxCompactArrays = 2 * 128 + 3;
// Slots per unit of a 4-byte array (tokens, positions, H2O totals): eight
// gathers per lane, so a sequence's few units spread over many warps
// instead of one warp walking all of them.
constexpr int kCompactSmallRows = 256;
constexpr int kMaxDepClasses = 3;        // distinct chunk sizes (K/V rows, H rows, 4-byte rows)

struct CompactArray {
  void *base;          // [batch][cap][row_bytes]
  int row_bytes;       // bulk arrays: multiple of 16; otherwise 4
  int bulk;            // rows moved by TMA bulk copies
  int rows_per_chunk;  // destination slots per unit
  int n_chunks;        // chunks per sequence = ceil(cap / rows_per_chunk) (upper bound of units)
  int dep_class;       // chunk-size class (index into the readers table)
  int paged;           // bulk K/V arrays of a paged cache: rows through CompactParams::pg
  int head_major;      // bulk K/V arrays [batch][Hkv][cap][row_bytes / Hkv]: a row is Hkv
                       // segments, one in each KV head's buffer
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
  int stage_bytes;            // shared-memory buffer of a unit (multiple of 128)
  int warps;                  // warps per CTA (each with two buffers)
  int ub_cached;              // unit_base is copied into shared memory after the buffers
                              // (n_arrays * batch + 1 entries fit): a unit's lookup of its
                              // (array, sequence) then costs no global round trips
  KvLayout pg;                // paged K/V arrays: pool row of logical slot (b, i)
  CompactArray arr[kMaxCompactArrays];
};

// Buffer size and warps per CTA for the largest row a cache moves (bytes);
// false when one row does not fit the shared-memory budget.
bool compact_shape(int max_row_bytes, int &stage_bytes, int &warps);
// Sets p.ub_cached when the unit table fits beside the staging buffers.
void compact_cache_units(CompactParams &p);
size_t compact_smem_bytes(const CompactParams &p);
// Launches the pre-passes and the (cooperative) compaction; `sms` = SM count.
cudaError_t launch_compact(const CompactParams &p, int sms, cudaStream_t st);

}  // namespace cc
