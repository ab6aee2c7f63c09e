// attn.cuh -- interface of the counter-causal attention kernel.
#pragma once
#include "cc_common.cuh"

namespace cc {

struct AttnParams {
  int batch, cap;
  int n_q_heads, n_kv_heads, head_dim, group;
  int P;                    // positions per work unit (attn_positions_per_unit(group))
  const int32_t *seq_len;   // device [batch]
  __nv_bfloat16 *out;       // row r, head t at out + r*out_ld + t*head_dim
  int out_ld;               // elements per output row (n_q_heads*head_dim, or twice that)
  int out_lo;               // > 0: also write lo = bf16(o - hi) at element offset out_lo
  int q_split;              // counter-causal, bf16 cache: Q rows are [hi | lo] bf16 pairs
                            // (the Q map spans 2 * n_q_heads heads, lo at head n_q_heads + t):
                            // S = Q_hi K^T + Q_lo K^T, and P enters P V as hi + lo too
  float scale_log2;         // log2(e) / sqrt(head_dim)
  int streams_per_group;    // unit order (set by launch_attention): see attn.cu
  int causal;               // 0: counter-causal (rows [0, n) attend (i, n)); 1: causal over
                            // the memory (rows [row_lo, n) attend [0, i], inference cycle)
  const int32_t *row_lo;    // causal: device [batch], first query slot of each sequence;
                            // counter-causal: null (rows from slot 0) or, with row_hi, the
                            // first row of a range
  const int32_t *row_hi;    // counter-causal: null (rows up to seq_len) or device [batch]:
                            // only rows [row_lo, row_hi) are computed, each still attending
                            // every later slot up to seq_len (cc_score_rows)
  int q_span;               // query slots per sequence at most (cap, or the chunk size)
  int kv_splits;            // > 1: each unit's key tiles split over kv_splits CTAs (few units)
  float *part_o;            // kv_splits > 1: [unit][split][256 rows][head_dim] unnormalised O
  float2 *part_ml;          // kv_splits > 1: [unit][split][256 rows] (reference max, row sum)
  const __nv_bfloat16 *q;   // decode kernel: Q [rows][Hq][dh]
  const void *k, *v;        // decode kernel: cache [rows][Hkv][dh] (bf16, or e4m3 bytes)
  int kv_fp8;               // decode kernel: K/V are e4m3 codes (the tile kernel takes bf16
                            // only: an e4m3 layer arrives as a bf16 copy of its codes); the
                            // K scale is folded into scale_log2 either way
  float v_scale;            // output = v_scale * (P V) / l (1 for a bf16 cache)
  int f16;                  // tile kernel, counter-causal, no split: Q, K, V, P and the
                            // output are fp16 (the fp16 operand mode of the scoring pass)
  KvLayout pg;              // paged K/V (pg.table nullptr: slot-major)
  int kv_rows;              // rows of the K/V tensor maps (a coordinate there reads zeros)
  unsigned *status;
};

constexpr int kDecMaxG = 8;   // query heads per KV head the decode kernel takes at most

int attn_positions_per_unit(int group);
// Work units of a launch (before key splits) and the partial-result floats
// per unit and split (kv_splits > 1).
long long attn_units(const AttnParams &p);
constexpr int kAttnPartRowFloats = 256;   // rows of a unit (times head_dim + 2 floats each)
// q: 3-D map over Q [rows][Hq][dh] (q_split: [rows][2 Hq][dh]), box {64, group, P}; k, v: 3-D maps over
// the cache [batch*cap][Hkv][dh] (bf16), box {64, 1, 128}; all 128-byte swizzled.
cudaError_t launch_attention(const CUtensorMap &q, const CUtensorMap &k, const CUtensorMap &v,
                             const AttnParams &p, cudaStream_t stream);
// Causal attention of one query row per sequence (q_span == 1, group <=
// kDecMaxG): CUDA-core kernel over kv_splits (>= 1) key ranges per unit, then
// the combine; needs q, k, v, part_o and part_ml.
cudaError_t launch_attention_decode(const AttnParams &p, cudaStream_t stream);

}  // namespace cc
