// gemv.cuh -- weight-streaming products of a few rows (the decode step of the
// inference cycle, one row per sequence): y = x W^T with W [N][K] bf16.
//
// With one to four rows the product is a matrix-vector stream bound by the
// weights' HBM bytes, so it is not shaped into tensor-core tiles.  A
// persistent CTA per SM takes a contiguous range of row groups (16 weight
// rows each); a producer warp streams them through a deep shared-memory ring
// with 2-D TMA copies (8 rows x 256 K-elements per box, two boxes per stage),
// and each of 16 consumer warps takes one weight row of every stage against
// the batch rows staged in shared memory.  A warp's row is one output, so no
// cross-warp sum is needed (deterministic results).  Epilogues match the tile
// GEMM's: RoPE'd bf16 (+bias), bf16 (+bias), fp32 residual add, SwiGLU and
// the argmax of the logits (one (max, column) pair per CTA).
#pragma once
#include "cc_common.cuh"

namespace cc {

enum GemvEpi : int {
  GEMV_ROPE = 0,       // out bf16 = RoPE(x W^T + bias); a group = 8 rotate-half column pairs
  GEMV_BF16 = 1,       // out bf16 = x W^T + bias; a group = 16 columns
  GEMV_RESID_F32 = 2,  // out fp32 += x W^T; a group = 16 columns
  GEMV_SWIGLU = 3,     // out bf16 = silu(x Wg^T) * (x Wu^T); a group = 8 columns
  GEMV_ARGMAX = 4,     // part[b][cta] = (largest logit of the CTA's columns, its first column)
};

constexpr int kGemvMaxRows = 4;
constexpr int kGemvConsumers = 16;   // consumer warps (one weight row of a stage each)
constexpr int kGemvMaxSegs = 3;
constexpr int kGemvBoxK = 256;       // K elements of one TMA box row (512 bytes)
constexpr int kGemvStageBytes = 2 * 8 * kGemvBoxK * 2;   // two boxes of 8 rows (one K chunk)
constexpr int kGemvMaxStages = 24;                       // K chunks the ring holds at most
// dynamic shared memory of one CTA at most (the 227 KB opt-in limit less the
// kernel's static shared memory)
constexpr size_t kGemvSmemMax = 226 * 1024;

struct GemvSeg {
  const __nv_bfloat16 *bias;  // ROPE, BF16: optional [N]
  void *out;                  // rows b*cap + slot, row stride ldo elements
  int ldo;
  int N, epi;
  int groups, group0;         // this segment's row groups: [group0, group0 + groups)
  int fp8;                    // ROPE, BF16: out is an e4m3 cache (bytes, value * qscale)
  float qscale;
  int kv_dest;                // ROPE, BF16: out holds K / V cache rows (through pg when paged)
};

struct GemvParams {
  GemvSeg seg[kGemvMaxSegs];
  int n_seg, n_groups, ctas, stages;
  int ks;                           // K chunks of 256 per ring stage (1, 2 or 4)
  const void *x;                    // rows b*cap + slot, row stride ldx elements
  int ldx, K;
  const __nv_bfloat16 *norm_gain;   // non-null: x is fp32 and the staged rows are
  float eps;                        //   bf16(x * gain / rms(x)) (the RMSNorm fused in)
  int batch, cap;
  const int32_t *row_lo, *row_hi;   // row of sequence b: slot row_lo[b] when row_hi[b] > row_lo[b]
  const int32_t *pos;               // ROPE: original positions [batch * cap]
  int head_dim;
  unsigned long long turns[64];     // ROPE: inv_freq_k / (2 pi) in 0.64 fixed point
  KvLayout pg;                      // paged cache rows of kv_dest segments
  float2 *part;                     // ARGMAX: [batch][part_ld], part_ld = ctas
  int part_ld;
  unsigned *status;
};

// The launch parameters: per segment the weights' tensor maps over [N][K],
// box {256, 8}, no swizzle (SwiGLU: the gate map, then the up map).
struct GemvLaunch {
  GemvParams p;
  CUtensorMap w[kGemvMaxSegs][2];
};

// Fills the segments' groups, the CTA count (at most `sms`), the stage size,
// the ring depth and part_ld.  Returns false when the staged rows leave no
// room for a ring of at least 3 stages.
bool gemv_plan(GemvParams &p, int sms);
size_t gemv_smem_bytes(const GemvParams &p);
cudaError_t launch_gemv(const GemvLaunch &l, cudaStream_t st);

}  // namespace cc
