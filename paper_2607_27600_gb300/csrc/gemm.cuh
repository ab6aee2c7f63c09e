// gemm.cuh -- interface of the tcgen05 GEMM with fused epilogues.
#pragma once
#include "cc_common.cuh"

namespace cc {

enum GemmEpi : int {
  EPI_F32 = 0,        // out fp32 [rows][ldo] = acc
  EPI_QROPE = 1,      // out bf16 [rows][ldo] = RoPE(acc) at pos[row], per head
  EPI_RESID_BF16 = 2, // out fp32 [rows][ldo] = acc + resid bf16 [rows][ld_resid]
  EPI_RESID_F32 = 3,  // out fp32 [rows][ldo] += acc
  EPI_SWIGLU = 4,     // out bf16 [rows][ldo] = silu(A Wg^T) * (A Wu^T)   (B = Wg, B2 = Wu)
  EPI_LSE = 5,        // out float2 [rows][ldo = n_tiles] = (max, sum exp) per vocab tile,
                      // z_target[row] = logit of tokens[row]
  EPI_BF16 = 6,       // out bf16 [rows][ldo] = acc (+ bias[col] if bias)
  EPI_QKV = 7,        // fused q/k/v projections (B = Wq, B2 = Wk, B3 = Wv, stacked by column
                      // tiles): Q RoPE'd to out, K RoPE'd to out_k, V to out_v
  EPI_ARGMAX = 8,     // greedy decoding, one valid row per sequence b: out float2
                      // [b][ldo = n_tiles] = (max, first column of the max) per column tile
  EPI_RESID_LOGIT = 9 // the last residual add fused with the logit head: x = out + acc
                      // (fp32 [rows][ldo], not stored back); head_part float2 [rows][n_tiles]
                      // = per column tile (sum x^2, sum x * head_gain * head_w[tokens[row]])
};

struct GemmParams {
  int batch, cap;
  const int32_t *seq_len;  // device [batch]: rows of sequence b end at slot seq_len[b]
  const int32_t *row_lo;   // device [batch] or nullptr: rows start at slot row_lo[b] (else 0)
  int N, K;
  int block_n;             // column tile width: 256, or 128 for narrow problems (not SwiGLU,
                           // LSE or the fused q/k/v projections)
  int n_tiles;             // column tiles (of block_n columns; SwiGLU: 128 outputs each)
  void *out;
  int ldo;
  const void *resid;
  int ld_resid;
  const int32_t *pos;      // EPI_QROPE
  const __nv_bfloat16 *bias;  // EPI_QROPE, EPI_BF16: optional per-column bias (before RoPE)
  int head_dim;            // EPI_QROPE
  const int32_t *tokens;   // EPI_LSE, EPI_RESID_LOGIT
  const __nv_bfloat16 *head_gain;   // EPI_RESID_LOGIT: final-norm gain [N]
  const __nv_bfloat16 *head_w;      // EPI_RESID_LOGIT: lm_head [vocab][N]
  int vocab;                        // EPI_RESID_LOGIT (tokens outside [0, vocab) read row 0)
  float2 *head_part;                // EPI_RESID_LOGIT: [rows][n_tiles]
  float *z_target;         // EPI_LSE
  // EPI_RESID_BF16 / EPI_RESID_F32 with norm_out: the next RMSNorm's input
  // is written too, unnormalised: norm_out bf16 [rows][ld_norm] = out * norm_gain
  // ([hi | lo] pairs, lo at column offset N, with norm_split), and
  // ss_part [rows][n_tiles] = the tile's partial sum of out^2
  __nv_bfloat16 *norm_out;
  const __nv_bfloat16 *norm_gain;
  int ld_norm, norm_split;
  float *ss_part;
  // EPI_SWIGLU / EPI_QROPE with row_ss: the A rows are unnormalised (as
  // above); the accumulators are scaled by rsqrt(sum_t row_ss[row][t] / ss_d
  // + eps), t < n_ss, before the activation (before the bias and RoPE)
  const float *row_ss;
  int n_ss, ss_d;
  float eps;
  unsigned *status;
  int a_split;             // A rows are [hi | lo] (2K values): D = hi W^T + lo W^T
  int raster;              // tile order: 0 = groups of `group` column tiles stay resident
                           // (B kept in L2, A streamed per group); 1 = groups of `group`
                           // row tiles stay resident (A kept, B streamed per group)
  int group;
  int pair;                // run as CTA pairs (256-column tiles, k_splits 1): the B tensor
                           // maps' boxes are 128 rows (each CTA loads half of a tile);
                           // raster 1 groups count pairs of row tiles
  int out_split;           // EPI_SWIGLU, EPI_QROPE (not into the cache): out rows are
                           // [hi | lo], lo at column offset N
  int ab_f16;              // A and W are fp16 (else bf16): the fp16 operand mode
  int out_f16;             // the activations written for the next product (EPI_SWIGLU and
                           // EPI_QROPE out, norm_out) are fp16 (not with the splits); a
                           // value above 65504 in magnitude sets CC_ERR_RANGE in status
  int k_splits;            // EPI_RESID_F32 / EPI_RESID_LOGIT only: K range split over
                           // k_splits work items per tile (< one wave of tiles); the splits
                           // add into out in order (EPI_RESID_LOGIT: the last one takes the
                           // partials instead)
  unsigned *split_flags;   // [tiles] (k_splits > 1): per-tile progress, epoch * 16 + split
  unsigned epoch;          // per-launch tag (>= 1) of split_flags values
  int n_q_tiles, n_k_tiles;   // EPI_QKV: column tiles of Q and of K (V has n_k_tiles too)
  void *out_k, *out_v;        // EPI_QKV: bf16 [rows][ldo_kv] destinations of K and V
  int ldo_kv;
  const __nv_bfloat16 *bias_k, *bias_v;   // EPI_QKV: optional biases of K and V
  int kv_dest;                // EPI_QROPE / EPI_BF16: the output is K / V cache rows (paged
                              // through pg; EPI_QKV: always for its K and V parts)
  KvLayout pg;                // paged K/V (pg.table nullptr: row b * cap + i)
  int kv_fp8;                 // EPI_QKV: K and V destinations are e4m3 (one byte each);
                              // EPI_QROPE / EPI_BF16: the destination is e4m3 K / V
  float k_qscale, v_qscale;   // kv_fp8: 1 / the K and V scales (code = rne(value * qscale))
  unsigned long long turns[64];  // EPI_QROPE: inv_freq_k / (2 pi) in 0.64 fixed point
};

int gemm_block_n(int epi);
int gemm_max_batch();
// a: A rows x K (box 64 x 128); b (and b2 for SwiGLU, b2 and b3 for the fused
// projections): weights N x K (box 64 x 256, or 64 x 128 for SwiGLU and for CTA pairs).
// grid: persistent CTAs (one per SM).
cudaError_t launch_gemm(int epi, const CUtensorMap &a, const CUtensorMap &b, const CUtensorMap &b2,
                        const CUtensorMap &b3, const GemmParams &p, int grid, cudaStream_t stream);

}  // namespace cc
