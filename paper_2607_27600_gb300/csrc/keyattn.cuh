// keyattn.cuh -- attention received by each cached key, with cached keys as
// proxy queries (the paper's importance and H2O comparison scorers, Sec. 4).
#pragma once
#include "cc_common.cuh"

namespace cc {

struct KeyAttnParams {
  int batch, cap, n_kv_heads, head_dim;
  const int32_t *seq_len;  // device [batch]: slots [0, n) are cached
  const int32_t *q_lo;     // device [batch] or nullptr: proxy queries are slots [q_lo, n)
  int recent;              // q_lo = max(0, n - recent) when q_lo == nullptr and recent > 0
  int q_span;              // proxy-query slots per sequence at most (sweep 0 unit count)
  int n_layers;            // layers in one launch (maps[0 .. n_layers))
  float *lse;              // [n_layers][batch][Hkv][ld]: log2-sum-exp of each proxy query
  float *part;             // [n_layers][batch][Hkv][ld]: per-head attention received by each key
  int ld;                  // cap rounded up to 128
  float scale_log2;        // log2(e) / sqrt(head_dim)
  KvLayout pg;             // paged K (pg.table nullptr: slot-major)
  int kv_rows;             // rows of the K tensor maps (a coordinate there reads zeros)
  unsigned *status;
};

constexpr int kKeyAttnMaxLayers = 64;

// The launch parameters: one 3-D tensor map per layer over its K cache
// [batch*cap][Hkv][dh], box {64, 1, 128} (all layers in one launch).
struct KeyAttnBatch {
  KeyAttnParams p;
  CUtensorMap k[kKeyAttnMaxLayers];
};

// Sweep 0 writes lse, sweep 1 (after it, same stream) writes part, for every layer.
cudaError_t launch_keyattn(const KeyAttnBatch &a, cudaStream_t st);
// out[b][j] (+)= sum over layers and KV heads of part[.][b][g][j] for j <
// seq_len[b] (fixed order); mean: divide by Hkv * (n - j) (importance);
// accumulate: add into out (H2O running total).
cudaError_t launch_keyattn_finish(const KeyAttnParams &p, float *out, bool mean, bool accumulate,
                                  cudaStream_t st);

// scores[b][j] = pos[b][j] (j < n), -inf past n
cudaError_t launch_recency_scores(const int32_t *pos, const int32_t *seq_len, int batch, int cap,
                                  float *scores, cudaStream_t st);
// scores = acc, +inf for the `recent` last slots, -inf past n
cudaError_t launch_h2o_scores(const float *acc, const int32_t *seq_len, int batch, int cap,
                              int recent, float *scores, cudaStream_t st);

}  // namespace cc
