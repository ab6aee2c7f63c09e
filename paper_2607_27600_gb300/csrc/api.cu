// api.cu -- the C ABI (include/cc.h, include/cc_kernels.h): argument checks,
// workspace layout, TMA tensor maps and the launch sequence of one refresh.
//
// Scoring pass per layer (Sec. 3.1, the standard pre-norm layer re-run under
// the counter-causal mask), on rows b*cap + i of a ragged batch:
//   xn = RMSNorm(h) ; Q = RoPE(xn Wq^T, pos)                 [rmsnorm, GEMM+RoPE]
//   O  = counter-causal attention(Q, K_l, V_l)               [attention]
//   h  = h + O Wo^T                                          [GEMM+residual]
//   xn = RMSNorm(h) ; A = silu(xn Wg^T) * (xn Wu^T)          [rmsnorm, GEMM+SwiGLU]
//   h  = h + A Wd^T                                          [GEMM+residual]
// then the head: -(final-norm(h) . W_U[x_i])  (logit mode, a gather-dot) or
// logsumexp(final-norm(h) W_U^T) - z[x_i]      (log-prob mode, GEMM+LSE).
#include <math.h>
#include <stdio.h>
#include <stdlib.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <mutex>

#include "attn.cuh"
#include "compact.cuh"
#include "gemm.cuh"
#include "gemv.cuh"
#include "keyattn.cuh"
#include "rowops.cuh"
#include "select.cuh"
#include "../../include/cc_kernels.h"
#include "../../include/cc_profile.h"
#include <vector>

namespace cc {

cudaError_t wait_kv_ready(const cc_kv_cache *kv, int l0, int l1, cudaStream_t st);
__device__ unsigned g_status_word;   // first device-side error since the last cc_get_status
}

namespace {

using namespace cc;

constexpr int kMaxDevices = 64;

// ---------------------------------------------------------------------------
// per-device state: status-word address, SM count
// ---------------------------------------------------------------------------
struct DevState {
  unsigned *status = nullptr;
  int sms = 0;
  bool ready = false;
};
DevState g_dev[kMaxDevices];
std::mutex g_mu;

bool dev_state(DevState **out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return false;
  std::lock_guard<std::mutex> lk(g_mu);
  DevState &d = g_dev[dev];
  if (!d.ready) {
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, cc::g_status_word) != cudaSuccess) return false;
    if (cudaDeviceGetAttribute(&d.sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return false;
    d.status = reinterpret_cast<unsigned *>(p);
    d.ready = true;
  }
  *out = &d;
  return true;
}

// ---------------------------------------------------------------------------
// optional launch timing (cc_profile.h)
// ---------------------------------------------------------------------------
struct TimingState {
  bool on = false;
  struct Rec { int kind; cudaEvent_t a, b; };
  std::vector<Rec> recs;
  std::vector<cudaEvent_t> pool;
  cudaEvent_t get() {
    if (!pool.empty()) { cudaEvent_t e = pool.back(); pool.pop_back(); return e; }
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    return e;
  }
};
TimingState g_timing;

// Brackets the launches issued in its scope with events on `st` when timing is on.
struct TimedScope {
  int kind;
  cudaStream_t st;
  cudaEvent_t a = nullptr;
  TimedScope(int k, cudaStream_t s) : kind(k), st(s) {
    if (g_timing.on && (a = g_timing.get())) cudaEventRecord(a, st);
  }
  ~TimedScope() {
    if (!a) return;
    cudaEvent_t b = g_timing.get();
    if (!b) { g_timing.pool.push_back(a); return; }
    cudaEventRecord(b, st);
    g_timing.recs.push_back({kind, a, b});
  }
};

// ---------------------------------------------------------------------------
// TMA tensor maps (driver entry point fetched through the runtime)
// ---------------------------------------------------------------------------
typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

// bf16 tensor of `rank` dims (dims[0] contiguous), strides in bytes for dims 1.., 128B swizzle.
bool make_tmap(CUtensorMap *m, const void *base, int rank, const uint64_t *dims,
               const uint64_t *strides, const uint32_t *box,
               CUtensorMapSwizzle swizzle = CU_TENSOR_MAP_SWIZZLE_128B,
               CUtensorMapDataType dtype = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t d[5], s[4];
  cuuint32_t bx[5], es[5];
  for (int i = 0; i < rank; ++i) {
    d[i] = dims[i];
    bx[i] = box[i];
    es[i] = 1;
    if (i > 0) s[i - 1] = strides[i - 1];
  }
  return fn(m, dtype, rank, const_cast<void *>(base), d, s, bx, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// rows x cols bf16 matrix (row pitch = cols), box 64 x box_rows
bool tmap_rows(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  const uint64_t dims[2] = {cols, rows};
  const uint64_t strides[1] = {cols * 2};
  const uint32_t box[2] = {64, box_rows};
  return make_tmap(m, base, 2, dims, strides, box);
}

// ---------------------------------------------------------------------------
// checks
// ---------------------------------------------------------------------------
bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

cc_status check_cfg(const cc_model_cfg *c) {
  if (!c) return CC_ERR_INVALID_ARG;
  if (c->n_layers < 1 || c->d_model < 1 || c->n_q_heads < 1 || c->n_kv_heads < 1 ||
      c->d_ff < 1 || c->vocab < 1 || !(c->rms_eps >= 0.f) || !(c->rope_theta > 0.f))
    return CC_ERR_INVALID_ARG;
  if (c->n_q_heads % c->n_kv_heads) return CC_ERR_INVALID_ARG;
  if (c->head_dim != 64 && c->head_dim != 128) return CC_ERR_UNSUPPORTED;
  if (c->d_model % 32 || c->d_ff % 32) return CC_ERR_UNSUPPORTED;
  if (c->n_q_heads / c->n_kv_heads > 256) return CC_ERR_UNSUPPORTED;
  if (c->rope_scaling_factor != 0.f &&
      !(c->rope_scaling_factor >= 1.f && c->rope_low_freq_factor > 0.f &&
        c->rope_high_freq_factor > c->rope_low_freq_factor && c->rope_original_max_pos > 0))
    return CC_ERR_INVALID_ARG;
  return CC_OK;
}

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

// Paging of the cache's K/V (table nullptr: slot-major [batch][cap]) and the
// rows of the K/V buffers (the pool, or batch * cap).
KvLayout kv_layout(const cc_model_cfg *c, const cc_kv_cache *kv) {
  KvLayout pg{};
  pg.hkv = c->n_kv_heads;
  pg.head_major = kv->kv_layout == CC_KV_HEAD_MAJOR ? 1 : 0;
  if (kv->block_table) {
    pg.table = kv->block_table;
    pg.page = kv->page_size;
    pg.pages_per_seq = kv->cap / kv->page_size;
    pg.n_pages = kv->n_pages;
  }
  return pg;
}
uint64_t kv_buffer_rows(const cc_kv_cache *kv) {
  return kv->block_table ? (uint64_t)kv->n_pages * kv->page_size : (uint64_t)kv->batch * kv->cap;
}

// Element format and layout of layer l's cached K/V.
struct KvFmt {
  bool fp8 = false;
  float k_scale = 1.f, v_scale = 1.f;
  KvLayout pg{};        // paged K/V (table nullptr: slot-major)
  uint64_t rows = 0;    // rows of the K/V buffers (0: batch * cap)
};
KvFmt kv_fmt(const cc_model_cfg *c, const cc_kv_cache *kv, int l) {
  KvFmt f;
  if (kv->kv_format == CC_KV_E4M3) {
    f.fp8 = true;
    f.k_scale = kv->kv_scale[2 * l];
    f.v_scale = kv->kv_scale[2 * l + 1];
  }
  f.pg = kv_layout(c, kv);
  f.rows = kv_buffer_rows(kv);
  return f;
}
int kv_elem_bytes(const cc_kv_cache *kv) { return kv->kv_format == CC_KV_E4M3 ? 1 : 2; }

// The cache's format fields: a known format; e4m3 needs finite positive
// scales for every layer.
bool kv_format_ok(const cc_model_cfg *c, const cc_kv_cache *kv) {
  if (kv->kv_layout != CC_KV_SLOT_MAJOR && kv->kv_layout != CC_KV_HEAD_MAJOR) return false;
  if (kv->kv_layout == CC_KV_HEAD_MAJOR && kv->block_table) return false;   // not paged
  if (kv->block_table) {   // pages of whole 128-slot key tiles that divide cap
    if (kv->page_size < 128 || kv->page_size % 128 || kv->cap % kv->page_size ||
        kv->n_pages < 1 || (uint64_t)kv->n_pages * kv->page_size >= (1ull << 31))
      return false;
  }
  if (kv->kv_format == CC_KV_BF16) return true;
  if (kv->kv_format != CC_KV_E4M3 || !kv->kv_scale) return false;
  for (int i = 0; i < 2 * c->n_layers; ++i)
    if (!(kv->kv_scale[i] > 0.f) || !std::isfinite(kv->kv_scale[i])) return false;
  return true;
}

struct ScoreWs {
  size_t xn, q, o, h, act, part, ztgt, hpart, sspart, flags, total;
  int n_vtiles;
  int n_htiles;   // column tiles of a d-column projection (at most d / 128): partials of
                  // the fused logit head (logit mode) and of the post-attention RMSNorm
};

// Per-tile progress flags of split-K GEMMs (at most one wave of tiles split).
constexpr int kSplitFlags = 1024;

// With CC_SCORE_PRECISE either pass carries the GEMM activations
// (normalised inputs, attention output, SwiGLU output) and the queries as
// [hi | lo] bf16 pairs: split = 2 copies per row.
ScoreWs score_layout(const cc_model_cfg *c, int batch, int cap, cc_score_mode mode, bool split_rows) {
  ScoreWs w{};
  const size_t R = (size_t)batch * cap;
  const size_t d = c->d_model, qd = (size_t)c->n_q_heads * c->head_dim, f = c->d_ff;
  const size_t split = split_rows ? 2 : 1;
  size_t off = 0;
  auto take = [&](size_t bytes) { size_t o = off; off = align256(off + bytes); return o; };
  w.xn = take(R * d * 2 * split);
  w.q = take(R * qd * 2 * split);
  w.o = take(R * qd * 2 * split);
  w.h = take(R * d * 4);
  w.act = take(R * f * 2 * split);
  w.n_vtiles = (c->vocab + 255) / 256;
  w.n_htiles = (int)((d + 127) / 128);
  if ((mode & 0xFF) == CC_SCORE_LOGPROB) {
    w.part = take(R * w.n_vtiles * 8);
    w.ztgt = take(R * 4);
  } else {
    w.hpart = take(R * w.n_htiles * 8);
  }
  w.sspart = take(R * w.n_htiles * 4);
  w.flags = take(kSplitFlags * 4);
  w.total = off;
  return w;
}

// RoPE: inv_freq_k / (2 pi) as 0.64 fixed point (angles reduced exactly on the device).
// With Llama-3.1 scaling, frequencies of long wavelengths are slowed by the
// factor, short ones kept, and the band between blended linearly in
// original_max_pos / wavelength.
void rope_turns(const cc_model_cfg *c, unsigned long long *turns) {
  const int half = c->head_dim / 2;
  for (int k = 0; k < half; ++k) {
    double inv_freq = pow((double)c->rope_theta, -2.0 * k / c->head_dim);
    if (c->rope_scaling_factor != 0.f) {
      const double f = c->rope_scaling_factor, lo = c->rope_low_freq_factor,
                   hi = c->rope_high_freq_factor, orig = c->rope_original_max_pos;
      const double wavelen = 2.0 * M_PI / inv_freq;
      if (wavelen > orig / lo) {
        inv_freq /= f;
      } else if (wavelen >= orig / hi) {
        const double a = (orig / wavelen - lo) / (hi - lo);
        inv_freq = (1.0 - a) * inv_freq / f + a * inv_freq;
      }
    }
    const double t = inv_freq / (2.0 * M_PI);   // < 1
    turns[k] = (unsigned long long)ldexp(t, 64);
  }
}

thread_local char g_last_error[256] = "";

cc_status cuda_fail(cudaError_t e, const char *what) {
  snprintf(g_last_error, sizeof(g_last_error), "%s: %s (%s)", what, cudaGetErrorName(e),
           cudaGetErrorString(e));
  return CC_ERR_CUDA;
}

cc_status tmap_fail() {
  snprintf(g_last_error, sizeof(g_last_error), "cuTensorMapEncodeTiled failed");
  return CC_ERR_CUDA;
}

cc_status device_fail() {
  cudaError_t e = cudaGetLastError();
  return cuda_fail(e, "device query (cudaGetDevice / cudaGetSymbolAddress)");
}

#define CC_TRY(expr)                                         \
  do {                                                       \
    cudaError_t e_ = (expr);                                 \
    if (e_ != cudaSuccess) return cuda_fail(e_, #expr);      \
  } while (0)

struct Gemm {
  CUtensorMap a, b, b2, b3;
  GemmParams p;
  uint64_t rows_est;   // rows visited at most (tile-count estimate on the host)
};

// One GEMM over the cache rows: A [R][K] (bf16 workspace) x W [N][K]^T.
// a_split: A rows are [hi | lo] (2K values) and the product is hi W^T + lo W^T.
// rows_hint: rows the GEMM visits at most (the traffic model's A size; 0 =
// every slot of the batch).
cc_status gemm_setup(Gemm &g, int epi, const void *A, int K, const void *W, const void *W2, int N,
                     int batch, int cap, const int32_t *seq_len, unsigned *status,
                     bool a_split = false, uint64_t rows_hint = 0) {
  const uint64_t R = (uint64_t)batch * cap;
  const uint64_t R_est = rows_hint ? rows_hint : R;
  int bn = gemm_block_n(epi);
  // narrow problems (less than one wave of 256-column tiles): 128-column
  // tiles double the tiles that share the SMs
  // (a residual GEMM long enough for two K splits keeps wide tiles and splits
  // K instead: plan_k_splits, measured faster for the down projection)
  const int nk_total = ((K + 63) / 64) * (a_split ? 2 : 1);
  const bool narrowable = epi == EPI_F32 || epi == EPI_QROPE || epi == EPI_RESID_BF16 ||
                          ((epi == EPI_RESID_F32 || epi == EPI_RESID_LOGIT) && nk_total < 128) ||
                          epi == EPI_BF16;
  DevState *dev_info = nullptr;
  const bool have_dev = dev_state(&dev_info);
  // CTA pairs: for launches of two waves or more of 128 x 256 tiles (a pair
  // takes two of them at once).  CC_GEMM_PAIRS=0: never; =2: whenever the
  // tiles are 256 columns wide (narrow problems keep wide tiles then)
  const char *pairs_env = getenv("CC_GEMM_PAIRS");
  const int pair_mode = !pairs_env ? 1 : pairs_env[0] == '0' ? 0 : pairs_env[0] == '2' ? 2 : 1;
  if (narrowable && have_dev && pair_mode != 2 &&
      ((R_est + 127) / 128) * (uint64_t)((N + 255) / 256) < (uint64_t)dev_info->sms)
    bn = 128;
  const bool pair = have_dev && epi != EPI_ARGMAX && (epi == EPI_SWIGLU || bn == 256) &&
                    (pair_mode == 2 ||
                     (pair_mode == 1 && ((R_est + 127) / 128) * (uint64_t)((N + bn - 1) / bn) >=
                                            2 * (uint64_t)dev_info->sms));
  if (!tmap_rows(&g.a, A, R, a_split ? 2 * K : K, 128)) return tmap_fail();
  if (!tmap_rows(&g.b, W, N, K, epi == EPI_SWIGLU || pair ? 128 : bn)) return tmap_fail();
  if (epi == EPI_SWIGLU) {
    if (!tmap_rows(&g.b2, W2, N, K, 128)) return tmap_fail();
  } else {
    g.b2 = g.b;
  }
  g.b3 = g.b;
  memset(&g.p, 0, sizeof(g.p));
  g.p.batch = batch;
  g.p.cap = cap;
  g.p.seq_len = seq_len;
  g.p.N = N;
  g.p.K = K;
  g.p.block_n = epi == EPI_SWIGLU ? 256 : bn;
  g.p.n_tiles = (N + bn - 1) / bn;
  g.p.status = status;
  g.p.a_split = a_split ? 1 : 0;
  // Tile order for L2 reuse: keep a slab of one operand resident (evict-last;
  // budget below) while the other streams past (evict-first; CTA pairs keep
  // both evict-last).  Weight slabs
  // resident (raster 0) is the default: a group's tiles of one activation row
  // tile run on consecutive CTAs, so the streamed row tile is read from DRAM
  // about once per group, and on the Llama-3-8B projections (K = 4096 and
  // 14336) this order measured 2-4 % faster than the activation-resident one
  // even where a count of whole-slab re-reads favoured the latter by up to
  // 16 %.  The activation-resident order is taken only when that count is
  // below 0.8x (an LM head whose weight is far larger than L2).
  const uint64_t R_used = R_est;
  // The slab budget: 40 MB, or 60 MB for an fp32-output GEMM whose streamed
  // activations outweigh its output (the down projection: each group of
  // resident weight tiles re-reads the activations).  Measured at the Llama-3-8B 16k launches (DRAM bytes read
  // per launch, 20 / 30 / 40 / 60 / 80 MB): the down projection (470 MB of
  // activations, 268 MB fp32 output) 5.5 / 3.6 / 3.8 / 2.6 / 3.2 GB, 1.06 ms
  // at 60 against 1.10 at 40; gate/up (134 MB in, 470 MB out) 3.2 / 2.4 /
  // 2.3 / 2.8 / 5.1 GB.
  const bool f32_out = epi == EPI_F32 || epi == EPI_RESID_BF16 || epi == EPI_RESID_F32 ||
                       epi == EPI_RESID_LOGIT;
  const double act_bytes = (double)R_used * K * (a_split ? 2.0 : 1.0) * 2;
  const double out_bytes = (double)R_used * N * (f32_out ? 4.0 : 2.0);
  const double budget = (f32_out && act_bytes > out_bytes ? 60.0 : 40.0) * (1 << 20);
  g.rows_est = R_used;
  const int num_m = (int)((R_used + 127) / 128), num_n = g.p.n_tiles;
  const double k_a = (a_split ? 2.0 : 1.0) * K;
  const int b_rows = epi == EPI_SWIGLU ? 256 : bn;   // weight rows of one column tile
  const double a_bytes = (double)R_used * k_a * 2, b_bytes = (double)num_n * b_rows * K * 2;
  const double a_slab = 128.0 * k_a * 2, b_slab = (double)b_rows * K * 2;
  const int gn = (int)std::max(1.0, std::min((double)num_n, floor(budget / b_slab)));
  const int gm = (int)std::max(1.0, std::min((double)num_m, floor(budget / a_slab)));
  const double t0 = b_bytes + a_bytes * ((num_n + gn - 1) / gn);
  const double t1 = a_bytes + b_bytes * ((num_m + gm - 1) / gm);
  g.p.raster = t1 < 0.8 * t0 ? 1 : 0;
  g.p.group = g.p.raster == 0 ? gn : gm;
  g.p.pair = pair ? 1 : 0;
  if (pair && g.p.raster == 1) g.p.group = std::max(1, gm / 2);   // pairs of row tiles
  return CC_OK;
}

// Fused q/k/v projections (one GEMM over the stacked weights [Wq; Wk; Wv]):
// possible when both q_dim and kv_dim are whole 256-column tiles.
bool qkv_fusable(const cc_model_cfg *c) {
  return (c->n_q_heads * c->head_dim) % 256 == 0 && (c->n_kv_heads * c->head_dim) % 256 == 0;
}

cc_status gemm_setup_qkv(Gemm &g, const void *xn, const cc_model_cfg *c,
                         const cc_layer_weights &lw, int batch, int cap, const int32_t *seq_len,
                         unsigned *status, uint64_t rows_hint) {
  const int d = c->d_model, qd = c->n_q_heads * c->head_dim, kvd = c->n_kv_heads * c->head_dim;
  cc_status s = gemm_setup(g, EPI_QKV, xn, d, lw.wq, nullptr, qd + 2 * kvd, batch, cap, seq_len,
                           status, false, rows_hint);
  if (s != CC_OK) return s;
  const uint32_t box = g.p.pair ? 128 : 256;   // a pair's CTAs load half a tile each
  if (!tmap_rows(&g.b, lw.wq, qd, d, box) || !tmap_rows(&g.b2, lw.wk, kvd, d, box) ||
      !tmap_rows(&g.b3, lw.wv, kvd, d, box))
    return tmap_fail();
  g.p.n_q_tiles = qd / 256;
  g.p.n_k_tiles = kvd / 256;
  g.p.ldo = qd;
  g.p.ldo_kv = kvd;
  g.p.bias = reinterpret_cast<const __nv_bfloat16 *>(lw.bq);
  g.p.bias_k = reinterpret_cast<const __nv_bfloat16 *>(lw.bk);
  g.p.bias_v = reinterpret_cast<const __nv_bfloat16 *>(lw.bv);
  g.p.head_dim = c->head_dim;
  rope_turns(c, g.p.turns);
  return CC_OK;
}

// K splits for a residual GEMM with less than one wave of output tiles
// (short caches): each split is a work item; splits add into the fp32
// residual in order (flags in the caller's workspace, tagged per launch).
void plan_k_splits(Gemm &g, int epi, int sms, unsigned *flags) {
  g.p.k_splits = 1;
  if ((epi != EPI_RESID_F32 && epi != EPI_RESID_LOGIT) || !flags || g.p.pair) return;
  const uint64_t tiles = ((g.rows_est + 127) / 128) * (uint64_t)g.p.n_tiles;
  const int nk_total = ((g.p.K + 63) / 64) * (g.p.a_split ? 2 : 1);
  if (tiles == 0 || tiles >= (uint64_t)sms || tiles > (uint64_t)kSplitFlags) return;
  // >= 64 k-blocks (K >= 4096) per split: shorter splits lose more to the
  // ordered epilogues than they gain (measured on Qwen2.5 O projections)
  int splits = std::min<int>((int)(sms / tiles), std::min(8, nk_total / 64));
  if (splits < 2) return;
  static std::atomic<unsigned> epoch{0};
  g.p.k_splits = splits;
  g.p.split_flags = flags;
  g.p.epoch = (epoch.fetch_add(1) % (1u << 27)) + 1;   // flags hold epoch * 16 + split
}

// Zeroes the split-K flags of a workspace once per call (a fresh workspace
// may hold any bits; later launches tag their values with new epochs).
cc_status clear_split_flags(unsigned *flags, cudaStream_t st) {
  CC_TRY(cudaMemsetAsync(flags, 0, kSplitFlags * 4, st));
  return CC_OK;
}

cc_status run_gemm(Gemm &g, int epi, int kind, int sms, cudaStream_t st) {
  TimedScope t(kind, st);
  CC_TRY(launch_gemm(epi, g.a, g.b, g.b2, g.b3, g.p, sms, st));
  return CC_OK;
}

// Key splits of the causal attention: at most this many (unit, split) CTAs
// write partial results, each split covering at least kAttnMinSplitTiles
// key tiles of 128.
constexpr int kAttnMaxSplitSlots = 160;
constexpr int kAttnMinSplitTiles = 4;

struct AttnPartials {
  float *o = nullptr;      // [kAttnMaxSplitSlots][256][head_dim]
  float2 *ml = nullptr;    // [kAttnMaxSplitSlots][256]
};

// Key splits for a launch of `units` CTAs: used when the units fill less
// than half of the SMs, so that a short chunk over a long memory (a decode
// step) still spreads its key tiles over the GPU.
int attn_key_splits(long long units, int cap, int sms) {
  if (units < 1 || units * 2 > sms) return 1;
  const long long by_tiles = ((long long)cap + 127) / 128 / kAttnMinSplitTiles;
  const long long s = std::min({(long long)sms / units, (long long)kAttnMaxSplitSlots / units,
                                by_tiles});
  return s >= 2 ? (int)s : 1;
}

// Key splits of the decode attention (one query row per unit): up to one
// CTA per SM in all, each split at least two chunks of 128 keys.
int attn_decode_splits(long long units, int cap, int sms) {
  const long long by_keys = std::max(1LL, ((long long)cap + 255) / 256);
  const long long s = std::min({std::max(1LL, (long long)sms / units),
                                std::max(1LL, (long long)kAttnMaxSplitSlots / units), by_keys});
  return (int)s;
}

// out: [R][Hq*dh] bf16, or with split [R][2*Hq*dh] = [hi | lo] per row.
// Counter-causal attention over rows [0, seq_len); with row_lo, the causal
// memory-augmented attention of the inference cycle over rows
// [row_lo, seq_len) (q_span: rows per sequence at most; with partials, key
// splits when the launch has few units).
cc_status run_attention(const cc_model_cfg *c, const void *q, const void *k, const void *v,
                        void *out, const int32_t *seq_len, int batch, int cap, unsigned *status,
                        cudaStream_t st, bool split = false, const int32_t *row_lo = nullptr,
                        int q_span = 0, const AttnPartials *parts = nullptr, int sms = 0,
                        KvFmt kvf = KvFmt(), bool q_split = false,
                        const int32_t *range_lo = nullptr, const int32_t *range_hi = nullptr,
                        void *kv_scratch = nullptr, size_t kv_scratch_bytes = 0,
                        bool f16 = false) {
  const int G = c->n_q_heads / c->n_kv_heads, dh = c->head_dim;
  const int P = attn_positions_per_unit(G);
  const uint64_t R = (uint64_t)batch * cap;
  if (q_split && row_lo) return CC_ERR_UNSUPPORTED;
  // fp16 operands (q and out fp16): the counter-causal pass with single operands
  if (f16 && (row_lo || split || q_split)) return CC_ERR_UNSUPPORTED;
  // one query row per sequence: the decode kernel, which reads either format
  const long long units0 = (long long)batch * c->n_kv_heads *
                           (((row_lo ? q_span : cap) + P - 1) / P);
  const bool decode = row_lo && q_span == 1 && G <= kDecMaxG && parts && parts->o && parts->ml &&
                      units0 <= kAttnMaxSplitSlots;
  if ((kvf.fp8 || f16) && !decode) {
    // the tile attention over an e4m3 cache, or with fp16 operands: the
    // layer's elements as bf16 or fp16 values (exact) in a slot-major scratch;
    // an e4m3 cache's scales stay folded into the softmax scale and the output
    // normalisation
    const size_t half = R * c->n_kv_heads * dh * 2;
    if (!kv_scratch || kv_scratch_bytes < 2 * half) return CC_ERR_UNSUPPORTED;
    uint8_t *ks = reinterpret_cast<uint8_t *>(kv_scratch);
    uint8_t *vs = ks + half;
    {
      TimedScope t(CC_KERNEL_KV_DEQUANT, st);
      CC_TRY(launch_kv_copy(reinterpret_cast<const uint8_t *>(k),
                            reinterpret_cast<const uint8_t *>(v), kvf.fp8, f16, kvf.pg, cap,
                            c->n_kv_heads, dh, seq_len, batch, ks, vs, status, st));
    }
    k = ks;
    v = vs;
    kvf.fp8 = false;
    kvf.pg = KvLayout{};
    kvf.pg.hkv = c->n_kv_heads;
    kvf.rows = R;
  }
  CUtensorMap tq, tk, tv;
  {
    // q_split: rows [hi heads | lo heads], the map spans both (lo at head Hq + t)
    const uint64_t qh = (uint64_t)c->n_q_heads * (q_split ? 2 : 1);
    const uint64_t dims[3] = {(uint64_t)dh, qh, R};
    const uint64_t strides[2] = {(uint64_t)dh * 2, qh * dh * 2};
    const uint32_t box[3] = {64, (uint32_t)G, (uint32_t)P};
    if (!make_tmap(&tq, q, 3, dims, strides, box)) return tmap_fail();
  }
  const uint64_t RK = kvf.rows ? kvf.rows : R;   // K/V buffer rows (paged: the pool)
  const bool hm = kvf.pg.head_major != 0;
  // slot-major maps (dh, Hkv, rows), box (.., 1, 128 slots); head-major maps
  // (dh, cap, batch*Hkv), box (.., 128 slots, 1): the same shared-memory image
  // (the tile kernel's maps: bf16; an e4m3 cache reaches here only for the
  // decode kernel, which reads the raw buffers)
  const uint64_t kv_dims[3] = {(uint64_t)dh, hm ? (uint64_t)cap : (uint64_t)c->n_kv_heads,
                               hm ? (uint64_t)batch * c->n_kv_heads : RK};
  const uint64_t kv_strides[2] = {(uint64_t)dh * 2,
                                  hm ? (uint64_t)cap * dh * 2 : (uint64_t)c->n_kv_heads * dh * 2};
  if (!kvf.fp8) {
    const uint32_t box[3] = {64, hm ? 128u : 1u, hm ? 1u : 128u};
    if (!make_tmap(&tk, k, 3, kv_dims, kv_strides, box)) return tmap_fail();
    if (!make_tmap(&tv, v, 3, kv_dims, kv_strides, box)) return tmap_fail();
  }
  AttnParams p{};
  p.batch = batch;
  p.cap = cap;
  p.n_q_heads = c->n_q_heads;
  p.n_kv_heads = c->n_kv_heads;
  p.head_dim = dh;
  p.group = G;
  p.P = P;
  p.seq_len = seq_len;
  p.out = reinterpret_cast<__nv_bfloat16 *>(out);
  p.out_ld = c->n_q_heads * dh * (split ? 2 : 1);
  p.out_lo = split ? c->n_q_heads * dh : 0;
  p.q_split = q_split ? 1 : 0;
  // e4m3 cache: S = Q . (codes * k_scale), so the K scale joins the softmax
  // scale; O = v_scale * P . codes, applied with the normalisation
  p.scale_log2 = (float)(1.4426950408889634 / sqrt((double)dh) * kvf.k_scale);
  p.kv_fp8 = kvf.fp8 ? 1 : 0;
  p.f16 = f16 ? 1 : 0;
  p.v_scale = kvf.v_scale;
  p.pg = kvf.pg;
  p.kv_rows = (int)RK;
  p.status = status;
  p.causal = row_lo ? 1 : 0;
  // counter-causal row range [range_lo, range_hi) (cc_score_rows); causal: row_lo
  p.row_lo = row_lo ? row_lo : range_lo;
  p.row_hi = row_lo ? nullptr : range_hi;
  p.q_span = row_lo ? q_span : cap;
  const long long units = attn_units(p);
  if (decode) {   // one query row per sequence: the decode kernel
    p.kv_splits = attn_decode_splits(units, cap, sms);
    p.part_o = parts->o;
    p.part_ml = parts->ml;
    p.q = reinterpret_cast<const __nv_bfloat16 *>(q);
    p.k = k;
    p.v = v;
    TimedScope t(CC_KERNEL_ATTN_CAUSAL, st);
    CC_TRY(launch_attention_decode(p, st));
    return CC_OK;
  }
  if (parts && parts->o && parts->ml) {
    p.kv_splits = attn_key_splits(attn_units(p), cap, sms);
    p.part_o = parts->o;
    p.part_ml = parts->ml;
  }
  TimedScope t(row_lo ? CC_KERNEL_ATTN_CAUSAL : CC_KERNEL_ATTENTION, st);
  CC_TRY(launch_attention(tq, tk, tv, p, st));
  return CC_OK;
}

// ---------------------------------------------------------------------------
// inference cycle, pre-fill: chunk append over the memory
// ---------------------------------------------------------------------------
struct AppendWs {
  ScoreWs s;          // xn, q, o, h, act rows b*cap + slot (the chunk's rows only are used)
  size_t lo, hi, part_o, part_ml, total;   // part_*: key-split partials of the attention
};

AppendWs append_layout(const cc_model_cfg *c, int batch, int cap) {
  AppendWs w{};
  w.s = score_layout(c, batch, cap, CC_SCORE_LOGIT, false);
  size_t off = w.s.total;
  w.lo = off;
  off = align256(off + (size_t)batch * 4);
  w.hi = off;
  off = align256(off + (size_t)batch * 4);
  w.part_o = off;
  off = align256(off + (size_t)kAttnMaxSplitSlots * 256 * c->head_dim * 4);
  w.part_ml = off;
  off = align256(off + (size_t)kAttnMaxSplitSlots * 256 * 8);
  w.total = off;
  return w;
}

// The tile attention over an e4m3 cache, or with fp16 operands, reads a
// 2-byte copy of the layer's K and V made in the activation buffer: whether
// it fits in `act_bytes` per slot.
bool kv_copy_fits(const cc_model_cfg *c, uint64_t act_bytes) {
  return 4ull * c->n_kv_heads * c->head_dim <= act_bytes;
}

cc_status check_append_args(const cc_model_cfg *c, const cc_model_weights *w,
                            const cc_kv_cache *kv, const int32_t *tokens_in,
                            const int32_t *count, int max_count, void *ws, size_t ws_bytes) {
  cc_status s = check_cfg(c);
  if (s != CC_OK) return s;
  if (!w || !kv || !w->layers || !w->embed || !kv->k || !kv->v || !tokens_in || max_count < 0 ||
      (!count && max_count != 1))   // no count array: one token each
    return CC_ERR_INVALID_ARG;
  if (kv->batch < 1 || kv->cap < 1 || !kv->seq_len || !kv->tokens || !kv->pos ||
      !kv_format_ok(c, kv))
    return CC_ERR_INVALID_ARG;
  if (kv->batch > gemm_max_batch()) return CC_ERR_UNSUPPORTED;
  if ((uint64_t)kv->batch * kv->cap >= (1ull << 31)) return CC_ERR_UNSUPPORTED;
  // an e4m3 layer copied for the tile attention (chunks, or query groups the
  // decode kernel does not take), checked before anything is enqueued
  const bool tile_attn = max_count != 1 || c->n_q_heads / c->n_kv_heads > kDecMaxG;
  if (kv->kv_format == CC_KV_E4M3 && tile_attn && !kv_copy_fits(c, 2ull * c->d_ff))
    return CC_ERR_UNSUPPORTED;
  for (int l = 0; l < c->n_layers; ++l) {
    const cc_layer_weights &lw = w->layers[l];
    const void *ptrs[] = {lw.attn_norm, lw.wq, lw.wk, lw.wv, lw.wo, lw.mlp_norm, lw.w_gate,
                          lw.w_up, lw.w_down, kv->k[l], kv->v[l]};
    for (const void *p : ptrs)
      if (!p || !aligned16(p)) return CC_ERR_INVALID_ARG;
    const void *opt[] = {lw.bq, lw.bk, lw.bv};
    for (const void *p : opt)
      if (p && !aligned16(p)) return CC_ERR_INVALID_ARG;
  }
  if (!aligned16(w->embed) || (kv->h_last && !aligned16(kv->h_last))) return CC_ERR_INVALID_ARG;
  if (!ws || !aligned16(ws) || ws_bytes < append_layout(c, kv->batch, kv->cap).total)
    return CC_ERR_WORKSPACE;
  return CC_OK;
}

// Decode-sized appends (one row per sequence, at most kGemvMaxRows
// sequences) run the layer products as weight-streaming GEMVs with the
// RMSNorms fused in: the tile GEMM would cover the weights with a few dozen
// CTAs for a single row.  Shared memory bounds the staged rows (K of every
// product, with the largest warp-partial buffer a plan can need).
bool gemv_decode_ok(const cc_model_cfg *c, int batch, int max_count) {
  if (max_count != 1 || batch < 1 || batch > kGemvMaxRows) return false;
  if (c->n_kv_heads * c->head_dim < 16 || c->vocab < 16) return false;   // 16 output rows at least
  const int ks[3] = {c->d_model, c->n_q_heads * c->head_dim, c->d_ff};
  for (int K : ks) {
    if (K < kGemvBoxK) return false;   // boxes no wider than the weights
    GemvParams p{};
    p.batch = batch;
    p.K = K;
    p.n_seg = 0;
    if (K % 8 || !gemv_plan(p, 1)) return false;
  }
  return true;
}

// One GEMV launch: up to three weight matrices (segments) over the same rows.
struct GemvCall {
  GemvLaunch l{};
  const void *w[kGemvMaxSegs][2] = {};
  void add(const void *w0, const void *w1, const void *bias, void *out, int ldo, int n, int epi) {
    GemvSeg &sg = l.p.seg[l.p.n_seg];
    sg = GemvSeg{};
    sg.bias = reinterpret_cast<const __nv_bfloat16 *>(bias);
    sg.out = out;
    sg.ldo = ldo;
    sg.N = n;
    sg.epi = epi;
    w[l.p.n_seg][0] = w0;
    w[l.p.n_seg][1] = w1;
    ++l.p.n_seg;
  }
};

GemvCall gemv_call(const cc_model_cfg *c, const cc_kv_cache *kv, const int32_t *lo,
                   const int32_t *hi, unsigned *status, const void *x, int ldx, int K,
                   const void *norm_gain) {
  GemvCall g;
  GemvParams &p = g.l.p;
  p.batch = kv->batch;
  p.cap = kv->cap;
  p.row_lo = lo;
  p.row_hi = hi;
  p.pos = kv->pos;
  p.head_dim = c->head_dim;
  p.eps = c->rms_eps;
  p.status = status;
  p.x = x;
  p.ldx = ldx;
  p.K = K;
  p.norm_gain = reinterpret_cast<const __nv_bfloat16 *>(norm_gain);
  rope_turns(c, p.turns);
  return g;
}

cc_status run_gemv(GemvCall &g, int kind, int sms, cudaStream_t st) {
  GemvParams &p = g.l.p;
  if (!gemv_plan(p, sms)) return CC_ERR_UNSUPPORTED;
  for (int s = 0; s < p.n_seg; ++s) {
    const uint64_t dims[2] = {(uint64_t)p.K, (uint64_t)p.seg[s].N};
    const uint64_t strides[1] = {(uint64_t)p.K * 2};
    const uint32_t box[2] = {(uint32_t)kGemvBoxK, 8};
    for (int j = 0; j < 2; ++j)
      if (g.w[s][j] && !make_tmap(&g.l.w[s][j], g.w[s][j], 2, dims, strides, box,
                                  CU_TENSOR_MAP_SWIZZLE_NONE))
        return tmap_fail();
  }
  TimedScope t(kind, st);
  CC_TRY(launch_gemv(g.l, st));
  return CC_OK;
}

cc_status run_append(const cc_model_cfg *c, const cc_model_weights *w, const cc_kv_cache *kv,
                     const int32_t *tokens_in, const int32_t *pos_in, const int32_t *count,
                     int max_count, void *ws, size_t ws_bytes, void *stream) {
  cc_status s = check_append_args(c, w, kv, tokens_in, count, max_count, ws, ws_bytes);
  if (s != CC_OK) return s;
  if (max_count == 0) return CC_OK;
  DevState *dev;
  if (!dev_state(&dev)) return device_fail();
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const int batch = kv->batch, cap = kv->cap, rows = batch * cap;
  const int d = c->d_model, qd = c->n_q_heads * c->head_dim, kvd = c->n_kv_heads * c->head_dim;
  const int f = c->d_ff;
  const AppendWs L = append_layout(c, batch, cap);
  uint8_t *wsb = reinterpret_cast<uint8_t *>(ws);
  void *xn = wsb + L.s.xn, *q = wsb + L.s.q, *o = wsb + L.s.o, *act = wsb + L.s.act;
  float *h = reinterpret_cast<float *>(wsb + L.s.h);
  int32_t *lo = reinterpret_cast<int32_t *>(wsb + L.lo), *hi = reinterpret_cast<int32_t *>(wsb + L.hi);
  unsigned *flags = reinterpret_cast<unsigned *>(wsb + L.s.flags);
  unsigned *status = dev->status;
  if ((s = clear_split_flags(flags, st)) != CC_OK) return s;
  const uint64_t used = (uint64_t)batch * max_count;   // rows the GEMMs visit at most
  AttnPartials parts;
  parts.o = reinterpret_cast<float *>(wsb + L.part_o);
  parts.ml = reinterpret_cast<float2 *>(wsb + L.part_ml);
  const bool use_gemv = gemv_decode_ok(c, batch, max_count);

  {
    TimedScope t(CC_KERNEL_APPEND, st);
    CC_TRY(launch_append_prepare(kv->seq_len, count, tokens_in, pos_in, max_count, kv->tokens,
                                 kv->pos, lo, hi, batch, cap, status, st));
  }
  {
    TimedScope t(CC_KERNEL_EMBED, st);
    CC_TRY(launch_embed(w->embed, kv->tokens, h, d, c->vocab, hi, cap, rows, status, st, lo,
                        max_count));
  }
  for (int l = 0; l < c->n_layers; ++l) {
    const cc_layer_weights &lw = w->layers[l];
    const KvFmt kvf = kv_fmt(c, kv, l);   // e4m3 cache: K/V rows written as codes of value / scale
    CC_TRY(wait_kv_ready(kv, l, l + 1, st));
    if (l == c->n_layers - 1 && kv->h_last) {   // H^(L-1), recorded for the fast approximation
      TimedScope t(CC_KERNEL_APPEND, st);
      CC_TRY(launch_store_bf16(h, kv->h_last, d, hi, lo, cap, rows, st, max_count));
    }
    if (use_gemv) {   // RMSNorm fused; q, k and v in one launch
      GemvCall g = gemv_call(c, kv, lo, hi, status, h, d, d, lw.attn_norm);
      g.add(lw.wq, nullptr, lw.bq, q, qd, qd, GEMV_ROPE);
      g.add(lw.wk, nullptr, lw.bk, kv->k[l], kvd, kvd, GEMV_ROPE);
      g.add(lw.wv, nullptr, lw.bv, kv->v[l], kvd, kvd, GEMV_BF16);
      for (int j = 1; j < 3; ++j) {   // K and V into the cache (e4m3 codes; paged rows)
        g.l.p.seg[j].fp8 = kvf.fp8 ? 1 : 0;
        g.l.p.seg[j].qscale = 1.f / (j == 1 ? kvf.k_scale : kvf.v_scale);
        g.l.p.seg[j].kv_dest = 1;
      }
      g.l.p.pg = kvf.pg;
      if ((s = run_gemv(g, CC_KERNEL_GEMM_QKV, dev->sms, st)) != CC_OK) return s;
    } else {
      TimedScope t(CC_KERNEL_RMSNORM, st);
      CC_TRY(launch_rmsnorm(h, true, lw.attn_norm, xn, d, c->rms_eps, hi, cap, rows, false, st, lo,
                            max_count));
    }
    // q = RoPE(xn Wq^T + bq) into the workspace; k = RoPE(xn Wk^T + bk) and
    // v = xn Wv^T + bv straight into the cache slots of the chunk
    if (!use_gemv && qkv_fusable(c)) {   // one GEMM over [Wq; Wk; Wv]
      Gemm g;
      if ((s = gemm_setup_qkv(g, xn, c, lw, batch, cap, hi, status, used)) != CC_OK) return s;
      g.p.row_lo = lo;
      g.p.out = q;
      g.p.out_k = kv->k[l];
      g.p.out_v = kv->v[l];
      g.p.pos = kv->pos;
      g.p.kv_fp8 = kvf.fp8 ? 1 : 0;
      g.p.k_qscale = 1.f / kvf.k_scale;
      g.p.v_qscale = 1.f / kvf.v_scale;
      g.p.pg = kvf.pg;
      if ((s = run_gemm(g, EPI_QKV, CC_KERNEL_GEMM_QKV, dev->sms, st)) != CC_OK) return s;
    }
    struct Proj { const void *w, *bias; void *out; int n, epi, kind; };
    const Proj projs[3] = {{lw.wq, lw.bq, q, qd, EPI_QROPE, CC_KERNEL_GEMM_QROPE},
                           {lw.wk, lw.bk, kv->k[l], kvd, EPI_QROPE, CC_KERNEL_GEMM_KV},
                           {lw.wv, lw.bv, kv->v[l], kvd, EPI_BF16, CC_KERNEL_GEMM_KV}};
    for (const Proj &pj : projs) {
      if (use_gemv || qkv_fusable(c)) break;
      Gemm g;
      if ((s = gemm_setup(g, pj.epi, xn, d, pj.w, nullptr, pj.n, batch, cap, hi, status, false,
                          used)) != CC_OK)
        return s;
      g.p.row_lo = lo;
      g.p.out = pj.out;
      g.p.ldo = pj.n;
      g.p.pos = kv->pos;
      g.p.bias = reinterpret_cast<const __nv_bfloat16 *>(pj.bias);
      g.p.head_dim = c->head_dim;
      if (pj.kind == CC_KERNEL_GEMM_KV) {   // K or V rows into the cache
        g.p.kv_dest = 1;
        g.p.pg = kvf.pg;
        g.p.kv_fp8 = kvf.fp8 ? 1 : 0;
        g.p.k_qscale = 1.f / kvf.k_scale;
        g.p.v_qscale = 1.f / kvf.v_scale;
      }
      if (pj.epi == EPI_QROPE) rope_turns(c, g.p.turns);
      if ((s = run_gemm(g, pj.epi, pj.kind, dev->sms, st)) != CC_OK) return s;
    }
    // o = attention of the chunk rows over the memory and the chunk (causal)
    // (act is free until the MLP: an e4m3 layer's bf16 copy for the tile attention)
    if ((s = run_attention(c, q, kv->k[l], kv->v[l], o, hi, batch, cap, status, st, false, lo,
                           max_count, &parts, dev->sms, kvf, false, nullptr, nullptr, act,
                           (size_t)batch * cap * c->d_ff * 2)) != CC_OK)
      return s;
    // h += o Wo^T; xn = RMSNorm(h); act = SwiGLU; h += act Wd^T
    if (use_gemv) {
      GemvCall go = gemv_call(c, kv, lo, hi, status, o, qd, qd, nullptr);
      go.add(lw.wo, nullptr, nullptr, h, d, d, GEMV_RESID_F32);
      if ((s = run_gemv(go, CC_KERNEL_GEMM_OPROJ, dev->sms, st)) != CC_OK) return s;
      GemvCall gu = gemv_call(c, kv, lo, hi, status, h, d, d, lw.mlp_norm);
      gu.add(lw.w_gate, lw.w_up, nullptr, act, f, f, GEMV_SWIGLU);
      if ((s = run_gemv(gu, CC_KERNEL_GEMM_GATEUP, dev->sms, st)) != CC_OK) return s;
      GemvCall gd = gemv_call(c, kv, lo, hi, status, act, f, f, nullptr);
      gd.add(lw.w_down, nullptr, nullptr, h, d, d, GEMV_RESID_F32);
      if ((s = run_gemv(gd, CC_KERNEL_GEMM_DOWN, dev->sms, st)) != CC_OK) return s;
      continue;
    }
    Gemm go;
    if ((s = gemm_setup(go, EPI_RESID_F32, o, qd, lw.wo, nullptr, d, batch, cap, hi, status,
                        false, used)) != CC_OK)
      return s;
    go.p.row_lo = lo;
    go.p.out = h;
    go.p.ldo = d;
    // the post-attention RMSNorm fused across the O and gate/up epilogues
    // (as in the scoring pass)
    float *ss_part = reinterpret_cast<float *>(wsb + L.s.sspart);
    go.p.norm_out = reinterpret_cast<__nv_bfloat16 *>(xn);
    go.p.norm_gain = reinterpret_cast<const __nv_bfloat16 *>(lw.mlp_norm);
    go.p.ld_norm = d;
    go.p.ss_part = ss_part;
    plan_k_splits(go, EPI_RESID_F32, dev->sms, flags);
    if ((s = run_gemm(go, EPI_RESID_F32, CC_KERNEL_GEMM_OPROJ, dev->sms, st)) != CC_OK) return s;
    Gemm gu;
    if ((s = gemm_setup(gu, EPI_SWIGLU, xn, d, lw.w_gate, lw.w_up, f, batch, cap, hi, status,
                        false, used)) != CC_OK)
      return s;
    gu.p.row_lo = lo;
    gu.p.out = act;
    gu.p.ldo = f;
    gu.p.row_ss = ss_part;
    gu.p.n_ss = go.p.n_tiles;
    gu.p.ss_d = d;
    gu.p.eps = c->rms_eps;
    if ((s = run_gemm(gu, EPI_SWIGLU, CC_KERNEL_GEMM_GATEUP, dev->sms, st)) != CC_OK) return s;
    Gemm gd;
    if ((s = gemm_setup(gd, EPI_RESID_F32, act, f, lw.w_down, nullptr, d, batch, cap, hi, status,
                        false, used)) != CC_OK)
      return s;
    gd.p.row_lo = lo;
    gd.p.out = h;
    gd.p.ldo = d;
    plan_k_splits(gd, EPI_RESID_F32, dev->sms, flags);
    if ((s = run_gemm(gd, EPI_RESID_F32, CC_KERNEL_GEMM_DOWN, dev->sms, st)) != CC_OK) return s;
  }
  {
    TimedScope t(CC_KERNEL_APPEND, st);
    CC_TRY(launch_append_finish(kv->seq_len, hi, batch, st));
  }
  return CC_OK;
}

cc_status check_score_args(const cc_model_cfg *c, const cc_model_weights *w, const cc_kv_cache *kv,
                           cc_score_mode mode, const float *scores, void *ws, size_t ws_bytes,
                           bool full) {
  cc_status s = check_cfg(c);
  if (s != CC_OK) return s;
  if (!w || !kv || !scores || !w->layers || !w->final_norm || !w->lm_head || !kv->k || !kv->v)
    return CC_ERR_INVALID_ARG;
  const int base_mode = mode & 0xFF;
  if ((base_mode != CC_SCORE_LOGIT && base_mode != CC_SCORE_LOGPROB) ||
      (mode & ~(0xFF | CC_SCORE_PRECISE | CC_SCORE_RANGE_ONLY | CC_SCORE_F16)) ||
      ((mode & CC_SCORE_PRECISE) && (mode & CC_SCORE_F16)))
    return CC_ERR_INVALID_ARG;
  if (kv->batch < 1 || kv->cap < 1 || !kv->seq_len || !kv->tokens || !kv->pos ||
      !kv_format_ok(c, kv))
    return CC_ERR_INVALID_ARG;
  if (kv->batch > gemm_max_batch()) return CC_ERR_UNSUPPORTED;
  if ((uint64_t)kv->batch * kv->cap >= (1ull << 31)) return CC_ERR_UNSUPPORTED;
  // the per-layer K/V copy of an e4m3 cache or of the fp16 mode, checked
  // before anything is enqueued
  if ((kv->kv_format == CC_KV_E4M3 || (mode & CC_SCORE_F16)) &&
      !kv_copy_fits(c, 2ull * c->d_ff * ((mode & CC_SCORE_PRECISE) ? 2 : 1)))
    return CC_ERR_UNSUPPORTED;
  if (full && !w->embed) return CC_ERR_INVALID_ARG;
  if (!full && !kv->h_last) return CC_ERR_INVALID_ARG;
  const int l0 = full ? 0 : c->n_layers - 1;
  for (int l = l0; l < c->n_layers; ++l) {
    const cc_layer_weights &lw = w->layers[l];
    const void *ptrs[] = {lw.attn_norm, lw.wq, lw.wo, lw.mlp_norm, lw.w_gate, lw.w_up, lw.w_down,
                          kv->k[l], kv->v[l]};
    for (const void *p : ptrs)
      if (!p || !aligned16(p)) return CC_ERR_INVALID_ARG;
    if (lw.bq && !aligned16(lw.bq)) return CC_ERR_INVALID_ARG;
  }
  const void *ptrs[] = {w->final_norm, w->lm_head, ws, kv->h_last, full ? w->embed : nullptr};
  for (const void *p : ptrs)
    if (p && !aligned16(p)) return CC_ERR_INVALID_ARG;
  if (!ws || ws_bytes < score_layout(c, kv->batch, kv->cap, mode, (mode & CC_SCORE_PRECISE) != 0).total)
    return CC_ERR_WORKSPACE;
  return CC_OK;
}

// rng_lo / rng_hi (device [batch], or both null): score only the rows
// [rng_lo[b], rng_hi[b]) of each sequence, each attending every later slot;
// every row kernel then visits those rows alone and the head writes only
// their scores (cc_score_rows), -inf elsewhere unless the mode has
// CC_SCORE_RANGE_ONLY (elsewhere untouched).
cc_status run_score(const cc_model_cfg *c, const cc_model_weights *w, const cc_kv_cache *kv,
                    cc_score_mode mode, float *scores, void *ws, size_t ws_bytes, void *stream,
                    bool full, const int32_t *rng_lo = nullptr, const int32_t *rng_hi = nullptr) {
  cc_status s = check_score_args(c, w, kv, mode, scores, ws, ws_bytes, full);
  if (s != CC_OK) return s;
  if ((rng_lo == nullptr) != (rng_hi == nullptr)) return CC_ERR_INVALID_ARG;
  DevState *dev;
  if (!dev_state(&dev)) return device_fail();
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const int batch = kv->batch, cap = kv->cap, rows = batch * cap;
  const int d = c->d_model, qd = c->n_q_heads * c->head_dim, f = c->d_ff;
  const bool split = (mode & CC_SCORE_PRECISE) != 0;   // [hi | lo] GEMM activations
  // [hi | lo] queries and attention probabilities too (an e4m3 cache's layers
  // enter the attention as exact bf16 copies)
  const bool split_q = split;
  // fp16 operands: the layer weights (the caller's), K/V (copied per layer),
  // the queries, P and the GEMM activations; the tensor maps are the same
  // (a tile copy moves 2-byte elements unchanged)
  const bool f16 = (mode & CC_SCORE_F16) != 0;
  const ScoreWs L = score_layout(c, batch, cap, mode, split);
  const bool logit = (mode & 0xFF) == CC_SCORE_LOGIT;
  const bool keep_outside = (mode & CC_SCORE_RANGE_ONLY) != 0;   // other entries untouched
  uint8_t *wsb = reinterpret_cast<uint8_t *>(ws);
  void *xn = wsb + L.xn, *q = wsb + L.q, *o = wsb + L.o, *act = wsb + L.act;
  float *h = reinterpret_cast<float *>(wsb + L.h);
  // the row kernels' row ends (the range's, or the sequence ends); attention
  // keys always run to the sequence end
  const int32_t *sl = rng_hi ? rng_hi : kv->seq_len;
  unsigned *status = dev->status;
  unsigned *flags = reinterpret_cast<unsigned *>(wsb + L.flags);
  if ((s = clear_split_flags(flags, st)) != CC_OK) return s;
  int n_htiles = 0;   // column tiles of the fused head's partials

  if (full) {
    TimedScope t(CC_KERNEL_EMBED, st);
    CC_TRY(launch_embed(w->embed, kv->tokens, h, d, c->vocab, sl, cap, rows, status, st, rng_lo));
  }
  const int l0 = full ? 0 : c->n_layers - 1;
  // per-column-tile partial sums of h^2 written by the residual GEMMs for the
  // next RMSNorm (the O projection's for the MLP norm, the down projection's
  // for the next layer's attention norm); each is read by the GEMM right
  // after its writer, before the next writer runs
  float *ss_part = reinterpret_cast<float *>(wsb + L.sspart);
  int ss_tiles = 0;   // column tiles of the attention norm's partials (0: none)
  for (int l = l0; l < c->n_layers; ++l) {
    const cc_layer_weights &lw = w->layers[l];
    const bool first_from_bf16 = !full;   // fast mode: the layer input is H^(L-1) (bf16)
    // xn = RMSNorm(h); after the first layer of the full pass the previous
    // down projection's epilogue has written xn = h * g (unnormalised) and
    // the partials, and the query projection scales its rows by 1 / rms(h)
    if (ss_tiles == 0) {
      TimedScope t(CC_KERNEL_RMSNORM, st);
      CC_TRY(launch_rmsnorm(first_from_bf16 ? kv->h_last : (const void *)h, !first_from_bf16,
                            lw.attn_norm, xn, d, c->rms_eps, sl, cap, rows, split, st, rng_lo, 0,
                            f16, status));
    }
    // Q = RoPE(xn Wq^T)
    Gemm gq;
    if ((s = gemm_setup(gq, EPI_QROPE, xn, d, lw.wq, nullptr, qd, batch, cap, sl, status,
                        split)) != CC_OK)
      return s;
    gq.p.row_lo = rng_lo;
    if (ss_tiles > 0) {
      gq.p.row_ss = ss_part;
      gq.p.n_ss = ss_tiles;
      gq.p.ss_d = d;
      gq.p.eps = c->rms_eps;
    }
    gq.p.out = q;
    gq.p.ldo = split_q ? 2 * qd : qd;
    gq.p.out_split = split_q ? 1 : 0;
    gq.p.ab_f16 = gq.p.out_f16 = f16 ? 1 : 0;
    gq.p.pos = kv->pos;
    gq.p.bias = reinterpret_cast<const __nv_bfloat16 *>(lw.bq);
    gq.p.head_dim = c->head_dim;
    rope_turns(c, gq.p.turns);
    if ((s = run_gemm(gq, EPI_QROPE, CC_KERNEL_GEMM_QROPE, dev->sms, st)) != CC_OK) return s;
    // O = counter-causal attention
    CC_TRY(wait_kv_ready(kv, l, l + 1, st));
    // (act is free until the MLP: the layer's bf16 copy of an e4m3 cache, or its
    // fp16 copy with fp16 operands, for the tile attention)
    if ((s = run_attention(c, q, kv->k[l], kv->v[l], o, kv->seq_len, batch, cap, status, st,
                           split, nullptr, 0, nullptr, 0, kv_fmt(c, kv, l), split_q, rng_lo,
                           rng_hi, act, (size_t)batch * cap * c->d_ff * 2 * (split ? 2 : 1),
                           f16)) != CC_OK)
      return s;
    // h = h + O Wo^T  (fast mode: h = H^(L-1) + O Wo^T)
    Gemm go;
    const int epi_o = first_from_bf16 ? EPI_RESID_BF16 : EPI_RESID_F32;
    if ((s = gemm_setup(go, epi_o, o, qd, lw.wo, nullptr, d, batch, cap, sl, status, split)) !=
        CC_OK)
      return s;
    go.p.row_lo = rng_lo;
    go.p.out = h;
    go.p.ldo = d;
    go.p.resid = kv->h_last;
    go.p.ld_resid = d;
    // the post-attention RMSNorm fused across the two GEMMs: this epilogue
    // writes xn = h * g (unnormalised) and per-tile sums of h^2; the gate/up
    // epilogue scales its accumulators by 1 / rms(h)
    go.p.norm_out = reinterpret_cast<__nv_bfloat16 *>(xn);
    go.p.norm_gain = reinterpret_cast<const __nv_bfloat16 *>(lw.mlp_norm);
    go.p.ld_norm = split ? 2 * d : d;
    go.p.norm_split = split ? 1 : 0;
    go.p.ss_part = ss_part;
    go.p.ab_f16 = go.p.out_f16 = f16 ? 1 : 0;
    plan_k_splits(go, epi_o, dev->sms, flags);
    if ((s = run_gemm(go, epi_o, CC_KERNEL_GEMM_OPROJ, dev->sms, st)) != CC_OK) return s;
    // act = silu(xn Wg^T / rms(h)) * (xn Wu^T / rms(h))
    Gemm gu;
    if ((s = gemm_setup(gu, EPI_SWIGLU, xn, d, lw.w_gate, lw.w_up, f, batch, cap, sl, status,
                        split)) != CC_OK)
      return s;
    gu.p.row_lo = rng_lo;
    gu.p.out = act;
    gu.p.ldo = split ? 2 * f : f;
    gu.p.out_split = split ? 1 : 0;
    gu.p.row_ss = ss_part;
    gu.p.n_ss = go.p.n_tiles;
    gu.p.ss_d = d;
    gu.p.eps = c->rms_eps;
    gu.p.ab_f16 = gu.p.out_f16 = f16 ? 1 : 0;
    if ((s = run_gemm(gu, EPI_SWIGLU, CC_KERNEL_GEMM_GATEUP, dev->sms, st)) != CC_OK) return s;
    // h = h + act Wd^T; in logit mode the last layer's add is fused with the
    // head: per column tile, partial sums of h^2 and of h * g . W_U[x_i]
    const int epi_d = logit && l == c->n_layers - 1 ? EPI_RESID_LOGIT : EPI_RESID_F32;
    Gemm gd;
    if ((s = gemm_setup(gd, epi_d, act, f, lw.w_down, nullptr, d, batch, cap, sl, status,
                        split)) != CC_OK)
      return s;
    gd.p.row_lo = rng_lo;
    gd.p.out = h;
    gd.p.ldo = d;
    gd.p.ab_f16 = gd.p.out_f16 = f16 ? 1 : 0;   // out_f16: the next layer's norm input
    if (epi_d == EPI_RESID_LOGIT) {
      gd.p.tokens = kv->tokens;
      gd.p.head_gain = reinterpret_cast<const __nv_bfloat16 *>(w->final_norm);
      gd.p.head_w = reinterpret_cast<const __nv_bfloat16 *>(w->lm_head);
      gd.p.vocab = c->vocab;
      gd.p.head_part = reinterpret_cast<float2 *>(wsb + L.hpart);
      n_htiles = gd.p.n_tiles;
    }
    ss_tiles = 0;
    if (full && l + 1 < c->n_layers) {   // the next layer's attention RMSNorm, fused as above
      gd.p.norm_out = reinterpret_cast<__nv_bfloat16 *>(xn);
      gd.p.norm_gain = reinterpret_cast<const __nv_bfloat16 *>(w->layers[l + 1].attn_norm);
      gd.p.ld_norm = split ? 2 * d : d;
      gd.p.norm_split = split ? 1 : 0;
      gd.p.ss_part = ss_part;
      ss_tiles = gd.p.n_tiles;
    }
    plan_k_splits(gd, epi_d, dev->sms, flags);
    if ((s = run_gemm(gd, epi_d, CC_KERNEL_GEMM_DOWN, dev->sms, st)) != CC_OK) return s;
  }
  // head
  if (logit) {
    TimedScope t(CC_KERNEL_HEAD_LOGIT, st);
    CC_TRY(launch_head_logit(reinterpret_cast<const float2 *>(wsb + L.hpart), n_htiles,
                             kv->tokens, scores, d, c->vocab, c->rms_eps, kv->seq_len, cap, rows,
                             status, st, rng_lo, rng_hi, keep_outside));
  } else {
    {
      TimedScope t(CC_KERNEL_RMSNORM, st);
      CC_TRY(launch_rmsnorm(h, true, w->final_norm, xn, d, c->rms_eps, sl, cap, rows, split, st,
                            rng_lo));
    }
    Gemm gl;
    if ((s = gemm_setup(gl, EPI_LSE, xn, d, w->lm_head, nullptr, c->vocab, batch, cap, sl,
                        status, split)) != CC_OK)
      return s;
    float2 *part = reinterpret_cast<float2 *>(wsb + L.part);
    float *zt = reinterpret_cast<float *>(wsb + L.ztgt);
    gl.p.row_lo = rng_lo;
    gl.p.out = part;
    gl.p.ldo = L.n_vtiles;
    gl.p.tokens = kv->tokens;
    gl.p.z_target = zt;
    if ((s = run_gemm(gl, EPI_LSE, CC_KERNEL_GEMM_LMHEAD, dev->sms, st)) != CC_OK) return s;
    TimedScope t(CC_KERNEL_LSE_COMBINE, st);
    CC_TRY(launch_lse_combine(part, L.n_vtiles, zt, scores, kv->seq_len, cap, rows, st, rng_lo,
                              rng_hi, keep_outside));
  }
  return CC_OK;
}

// compaction plan: arrays and unit counts
// Compaction workspace: unit_base table | flags (zeroed per call) | readers table (-1 per call)
struct CompactPlan {
  CompactParams p;
  size_t base_bytes, flags_bytes, deps_bytes, ws_bytes;
};

int g_withhold_unit = -1;   // cc_debug_withhold_compact_unit: consumed by the next cc_compact_kv

cc_status compact_plan(const cc_model_cfg *c, const cc_kv_cache *kv, CompactPlan &plan) {
  cc_status s = check_cfg(c);
  if (s != CC_OK) return s;
  if (!kv || kv->batch < 1 || kv->cap < 1 || !kv->k || !kv->v || !kv->tokens || !kv->pos ||
      !kv->seq_len || !kv_format_ok(c, kv))
    return CC_ERR_INVALID_ARG;
  CompactParams &p = plan.p;
  memset(&p, 0, sizeof(p));
  p.withhold_unit = -1;
  p.batch = kv->batch;
  p.cap = kv->cap;
  int n = 0, units = 0;
  auto class_of = [&](int rows) -> int {
    for (int c = 0; c < p.n_classes; ++c)
      if (p.class_rows[c] == rows) return c;
    if (p.n_classes >= kMaxDepClasses) return -1;
    p.class_rows[p.n_classes] = rows;
    p.class_chunks[p.n_classes] = (kv->cap + rows - 1) / rows;
    return p.n_classes++;
  };
  auto add = [&](void *base, int row_bytes, bool bulk, bool paged = false,
                 bool head_major = false) -> bool {
    if (!base) return true;
    if (n >= kMaxCompactArrays || !aligned16(base)) return false;
    CompactArray &A = p.arr[n++];
    A.base = base;
    A.row_bytes = row_bytes;
    A.bulk = bulk ? 1 : 0;
    A.paged = paged ? 1 : 0;
    A.head_major = head_major ? 1 : 0;
    A.rows_per_chunk = bulk ? (row_bytes <= p.stage_bytes ? p.stage_bytes / row_bytes : 0)
                            : std::min(kCompactSmallRows, p.stage_bytes / 4);
    if (A.rows_per_chunk < 1) return false;
    A.n_chunks = (kv->cap + A.rows_per_chunk - 1) / A.rows_per_chunk;
    A.dep_class = class_of(A.rows_per_chunk);
    if (A.dep_class < 0) return false;
    units += kv->batch * A.n_chunks;
    return true;
  };
  const int kv_row = c->n_kv_heads * c->head_dim * kv_elem_bytes(kv);
  // staging shape of the copy kernel for the largest row moved
  const int max_row = std::max(kv_row, kv->h_last ? c->d_model * 2 : 0);
  if (!compact_shape(max_row, p.stage_bytes, p.warps)) return CC_ERR_UNSUPPORTED;
  p.pg = kv_layout(c, kv);   // K/V rows through the block table when paged
  const bool paged = kv->block_table != nullptr;
  const bool hm = kv->kv_layout == CC_KV_HEAD_MAJOR;   // rows of Hkv segments
  // the 4-byte arrays first: their gathers then overlap the bulk copies
  // instead of trailing them (units run in ascending order)
  if (!add(kv->tokens, 4, false) || !add(kv->pos, 4, false)) return CC_ERR_INVALID_ARG;
  if (!add(kv->h2o_acc, 4, false)) return CC_ERR_INVALID_ARG;   // comparison scorer totals
  for (int l = 0; l < c->n_layers; ++l) {
    if (!add(kv->k[l], kv_row, true, paged, hm) || !add(kv->v[l], kv_row, true, paged, hm))
      return CC_ERR_UNSUPPORTED;
  }
  if (!add(kv->h_last, c->d_model * 2, true)) return CC_ERR_UNSUPPORTED;
  p.n_arrays = n;
  p.total_units = units;
  if (n < 2 || units < 2) return CC_ERR_INVALID_ARG;   // tokens and pos are always compacted
  compact_cache_units(p);
  size_t deps_entries = 0;
  for (int c = 0; c < p.n_classes; ++c) {
    p.class_offset[c] = (long long)deps_entries;
    deps_entries += (size_t)kv->batch * p.class_chunks[c];
  }
  plan.base_bytes = align256(((size_t)n * kv->batch + 1) * sizeof(int));
  plan.flags_bytes = align256((size_t)units * 4);
  plan.deps_bytes = align256(deps_entries * sizeof(int2));
  plan.ws_bytes = plan.base_bytes + plan.flags_bytes + plan.deps_bytes;
  return CC_OK;
}

// Points the plan at workspace `ws` and clears what must start cleared.
cc_status compact_bind(CompactPlan &plan, void *ws, cudaStream_t st) {
  uint8_t *w = reinterpret_cast<uint8_t *>(ws);
  plan.p.unit_base = reinterpret_cast<int *>(w);
  plan.p.flags = reinterpret_cast<unsigned *>(w + plan.base_bytes);
  plan.p.deps = reinterpret_cast<int2 *>(w + plan.base_bytes + plan.flags_bytes);
  CC_TRY(cudaMemsetAsync(plan.p.flags, 0, plan.flags_bytes, st));
  CC_TRY(cudaMemsetAsync(plan.p.deps, 0xFF, plan.deps_bytes, st));
  return CC_OK;
}

}  // namespace

// ===========================================================================
// C ABI
// ===========================================================================
extern "C" {

// ---- the paper's comparison scorers (Sec. 4) ---------------------------------
cc_status cc_score_recency(const cc_kv_cache *kv, float *scores, void *stream) {
  if (!kv || !scores || !kv->pos || !kv->seq_len || kv->batch < 1 || kv->cap < 1)
    return CC_ERR_INVALID_ARG;
  CC_TRY(launch_recency_scores(kv->pos, kv->seq_len, kv->batch, kv->cap, scores,
                               reinterpret_cast<cudaStream_t>(stream)));
  return CC_OK;
}

size_t cc_keyattn_workspace_size(const cc_model_cfg *cfg, int32_t batch, int32_t cap) {
  if (check_cfg(cfg) != CC_OK || batch < 1 || cap < 1) return 0;
  if (cfg->n_layers > kKeyAttnMaxLayers) return 0;
  const size_t ld = ((size_t)cap + 127) / 128 * 128;
  // lse2 and per-head sums of every layer (H2O runs all layers in one launch)
  return 2 * (size_t)cfg->n_layers * batch * cfg->n_kv_heads * ld * 4;
}

// Sweeps over layers [l0, l1) in one launch each; out = finish(part)
// (mean: importance; accumulate: H2O).
cc_status run_keyattn(const cc_model_cfg *c, const cc_kv_cache *kv, int l0, int l1, int recent,
                      float *out, bool mean, bool accumulate, void *ws, cudaStream_t st,
                      unsigned *status) {
  const int batch = kv->batch, cap = kv->cap, dh = c->head_dim;
  const uint64_t R = (uint64_t)batch * cap;
  static KeyAttnBatch a;   // ~8 KB: kept off the stack; guarded below
  static std::mutex mu;
  std::lock_guard<std::mutex> lk(mu);
  memset(&a, 0, sizeof(a));
  const uint64_t RK = kv_buffer_rows(kv);   // K buffer rows (paged: the pool)
  (void)R;
  const bool hm = kv->kv_layout == CC_KV_HEAD_MAJOR;   // see run_attention
  const uint64_t dims[3] = {(uint64_t)dh, hm ? (uint64_t)cap : (uint64_t)c->n_kv_heads,
                            hm ? (uint64_t)batch * c->n_kv_heads : RK};
  const uint64_t strides[2] = {(uint64_t)dh * 2,
                               hm ? (uint64_t)cap * dh * 2 : (uint64_t)c->n_kv_heads * dh * 2};
  const uint32_t box[3] = {64, hm ? 128u : 1u, hm ? 1u : 128u};
  for (int l = l0; l < l1; ++l)
    if (!make_tmap(&a.k[l - l0], kv->k[l], 3, dims, strides, box)) return tmap_fail();
  KeyAttnParams &p = a.p;
  p.pg = kv_layout(c, kv);
  p.kv_rows = (int)RK;
  p.batch = batch;
  p.cap = cap;
  p.n_kv_heads = c->n_kv_heads;
  p.head_dim = dh;
  p.seq_len = kv->seq_len;
  p.q_lo = nullptr;
  p.recent = recent;
  p.q_span = recent > 0 ? std::min(recent, cap) : cap;
  p.n_layers = l1 - l0;
  p.ld = (cap + 127) / 128 * 128;
  p.lse = reinterpret_cast<float *>(ws);
  p.part = p.lse + (size_t)p.n_layers * batch * c->n_kv_heads * p.ld;
  p.scale_log2 = (float)(1.4426950408889634 / sqrt((double)dh));
  p.status = status;
  CC_TRY(wait_kv_ready(kv, l0, l1, st));
  TimedScope t(CC_KERNEL_KEYATTN, st);
  CC_TRY(launch_keyattn(a, st));
  CC_TRY(launch_keyattn_finish(p, out, mean, accumulate, st));
  return CC_OK;
}

cc_status check_keyattn_args(const cc_model_cfg *c, const cc_kv_cache *kv, void *ws,
                             size_t ws_bytes, int l0) {
  cc_status s = check_cfg(c);
  if (s != CC_OK) return s;
  if (!kv || !kv->k || !kv->seq_len || kv->batch < 1 || kv->cap < 1) return CC_ERR_INVALID_ARG;
  if ((uint64_t)kv->batch * kv->cap >= (1ull << 31)) return CC_ERR_UNSUPPORTED;
  if (c->n_layers > kKeyAttnMaxLayers) return CC_ERR_UNSUPPORTED;
  if (kv->kv_format != CC_KV_BF16) return CC_ERR_UNSUPPORTED;   // bf16 keys only
  if (!kv_format_ok(c, kv)) return CC_ERR_INVALID_ARG;
  for (int l = l0; l < c->n_layers; ++l)
    if (!kv->k[l] || !aligned16(kv->k[l])) return CC_ERR_INVALID_ARG;
  if (!ws || !aligned16(ws) || ws_bytes < cc_keyattn_workspace_size(c, kv->batch, kv->cap))
    return CC_ERR_WORKSPACE;
  return CC_OK;
}

cc_status cc_score_importance(const cc_model_cfg *cfg, const cc_kv_cache *kv, float *scores,
                              void *ws, size_t ws_bytes, void *stream) {
  cc_status s = check_keyattn_args(cfg, kv, ws, ws_bytes, cfg ? cfg->n_layers - 1 : 0);
  if (s != CC_OK) return s;
  if (!scores) return CC_ERR_INVALID_ARG;
  DevState *dev;
  if (!dev_state(&dev)) return device_fail();
  return run_keyattn(cfg, kv, cfg->n_layers - 1, cfg->n_layers, 0, scores, true, false, ws,
                     reinterpret_cast<cudaStream_t>(stream), dev->status);
}

cc_status cc_h2o_accumulate(const cc_model_cfg *cfg, const cc_kv_cache *kv, int32_t recent,
                            void *ws, size_t ws_bytes, void *stream) {
  cc_status s = check_keyattn_args(cfg, kv, ws, ws_bytes, 0);
  if (s != CC_OK) return s;
  if (!kv->h2o_acc || recent < 1) return CC_ERR_INVALID_ARG;
  DevState *dev;
  if (!dev_state(&dev)) return device_fail();
  return run_keyattn(cfg, kv, 0, cfg->n_layers, recent, kv->h2o_acc, false, true, ws,
                     reinterpret_cast<cudaStream_t>(stream), dev->status);
}

cc_status cc_score_h2o(const cc_kv_cache *kv, int32_t recent, float *scores, void *stream) {
  if (!kv || !scores || !kv->h2o_acc || !kv->seq_len || kv->batch < 1 || kv->cap < 1 || recent < 0)
    return CC_ERR_INVALID_ARG;
  CC_TRY(launch_h2o_scores(kv->h2o_acc, kv->seq_len, kv->batch, kv->cap, recent, scores,
                           reinterpret_cast<cudaStream_t>(stream)));
  return CC_OK;
}

// ---- decode step (greedy): append one token each, LM head, argmax -------------
constexpr int kDecodeMinParts = 1024;   // argmax pairs per sequence the workspace holds at least

size_t decode_part_offset(const cc_model_cfg *c, int batch, int cap) {
  return align256(append_layout(c, batch, cap).total);
}

size_t cc_decode_workspace_size(const cc_model_cfg *cfg, int32_t batch, int32_t cap) {
  if (check_cfg(cfg) != CC_OK || batch < 1 || cap < 1) return 0;
  // (max, column) pairs per sequence: one per LM-head column tile of either
  // width, or one per CTA of the weight-streaming LM head
  const size_t n_tiles = std::max<size_t>(((size_t)cfg->vocab + 127) / 128, kDecodeMinParts);
  return decode_part_offset(cfg, batch, cap) + align256((size_t)batch * n_tiles * 8);
}

cc_status cc_decode_step(const cc_model_cfg *cfg, const cc_model_weights *w,
                         const cc_kv_cache *cache, const int32_t *tokens_in, int32_t *next_tokens,
                         float *next_logit, void *ws, size_t ws_bytes, void *stream) {
  if (!cfg || !w || !cache || !tokens_in || !next_tokens || !w->final_norm || !w->lm_head)
    return CC_ERR_INVALID_ARG;
  if (check_cfg(cfg) != CC_OK) return check_cfg(cfg);
  if (!aligned16(w->final_norm) || !aligned16(w->lm_head)) return CC_ERR_INVALID_ARG;
  if (!ws || ws_bytes < cc_decode_workspace_size(cfg, cache->batch, cache->cap))
    return CC_ERR_WORKSPACE;
  cc_status s = run_append(cfg, w, cache, tokens_in, nullptr, nullptr, 1, ws, ws_bytes, stream);
  if (s != CC_OK) return s;
  DevState *dev;
  if (!dev_state(&dev)) return device_fail();
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const int batch = cache->batch, cap = cache->cap, d = cfg->d_model;
  const AppendWs L = append_layout(cfg, batch, cap);
  uint8_t *wsb = reinterpret_cast<uint8_t *>(ws);
  void *xn = wsb + L.s.xn;
  float *h = reinterpret_cast<float *>(wsb + L.s.h);
  int32_t *lo = reinterpret_cast<int32_t *>(wsb + L.lo), *hi = reinterpret_cast<int32_t *>(wsb + L.hi);
  float2 *part = reinterpret_cast<float2 *>(wsb + decode_part_offset(cfg, batch, cap));
  if (gemv_decode_ok(cfg, batch, 1) && dev->sms <= kDecodeMinParts) {
    // final norm fused; one (max, first column) pair per CTA
    GemvCall g = gemv_call(cfg, cache, lo, hi, dev->status, h, d, d, w->final_norm);
    g.add(w->lm_head, nullptr, nullptr, nullptr, 0, cfg->vocab, GEMV_ARGMAX);
    g.l.p.part = part;
    if ((s = run_gemv(g, CC_KERNEL_GEMM_LMHEAD, dev->sms, st)) != CC_OK) return s;
    TimedScope t(CC_KERNEL_APPEND, st);
    CC_TRY(launch_argmax_combine(part, g.l.p.part_ld, lo, hi, batch, next_tokens, next_logit, st));
    return CC_OK;
  }
  {
    TimedScope t(CC_KERNEL_RMSNORM, st);
    CC_TRY(launch_rmsnorm(h, true, w->final_norm, xn, d, cfg->rms_eps, hi, cap, batch * cap, false,
                          st, lo, 1));
  }
  Gemm g;
  if ((s = gemm_setup(g, EPI_ARGMAX, xn, d, w->lm_head, nullptr, cfg->vocab, batch, cap, hi,
                      dev->status, false, (uint64_t)batch)) != CC_OK)
    return s;
  g.p.row_lo = lo;
  g.p.out = part;
  g.p.ldo = g.p.n_tiles;
  if ((s = run_gemm(g, EPI_ARGMAX, CC_KERNEL_GEMM_LMHEAD, dev->sms, st)) != CC_OK) return s;
  {
    TimedScope t(CC_KERNEL_APPEND, st);
    CC_TRY(launch_argmax_combine(part, g.p.n_tiles, lo, hi, batch, next_tokens, next_logit, st));
  }
  return CC_OK;
}

size_t cc_append_workspace_size(const cc_model_cfg *cfg, int32_t batch, int32_t cap) {
  if (check_cfg(cfg) != CC_OK || batch < 1 || cap < 1) return 0;
  return append_layout(cfg, batch, cap).total;
}

cc_status cc_append_chunk(const cc_model_cfg *cfg, const cc_model_weights *w,
                          const cc_kv_cache *cache, const int32_t *tokens_in,
                          const int32_t *pos_in, const int32_t *count, int32_t max_count,
                          void *ws, size_t ws_bytes, void *stream) {
  return run_append(cfg, w, cache, tokens_in, pos_in, count, max_count, ws, ws_bytes, stream);
}

size_t cc_score_workspace_size(const cc_model_cfg *cfg, int32_t batch, int32_t cap,
                               cc_score_mode mode) {
  if (check_cfg(cfg) != CC_OK || batch < 1 || cap < 1) return 0;
  return score_layout(cfg, batch, cap, mode, (mode & CC_SCORE_PRECISE) != 0).total;
}

cc_status cc_score_layer(const cc_model_cfg *cfg, const cc_model_weights *w,
                         const cc_kv_cache *cache, cc_score_mode mode, float *scores, void *ws,
                         size_t ws_bytes, void *stream) {
  return run_score(cfg, w, cache, mode, scores, ws, ws_bytes, stream, false);
}

cc_status cc_score_full(const cc_model_cfg *cfg, const cc_model_weights *w,
                        const cc_kv_cache *cache, cc_score_mode mode, float *scores, void *ws,
                        size_t ws_bytes, void *stream) {
  return run_score(cfg, w, cache, mode, scores, ws, ws_bytes, stream, true);
}

cc_status cc_bf16_to_f16(const void *src, void *dst, size_t n, void *stream) {
  if (n == 0) return CC_OK;
  if (!src || !dst || n % 8 || !aligned16(src) || !aligned16(dst)) return CC_ERR_INVALID_ARG;
  const uintptr_t a = reinterpret_cast<uintptr_t>(src), b = reinterpret_cast<uintptr_t>(dst);
  if (a < b + 2 * n && b < a + 2 * n) return CC_ERR_INVALID_ARG;   // overlapping
  DevState *dev;
  if (!dev_state(&dev)) return device_fail();
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  TimedScope t(CC_KERNEL_OTHER, st);
  CC_TRY(launch_bf16_to_f16(src, dst, n, dev->sms, dev->status, st));
  return CC_OK;
}

cc_status cc_score_rows(const cc_model_cfg *cfg, const cc_model_weights *w,
                        const cc_kv_cache *cache, cc_score_mode mode, int32_t full,
                        const int32_t *row_lo, const int32_t *row_hi, float *scores, void *ws,
                        size_t ws_bytes, void *stream) {
  return run_score(cfg, w, cache, mode, scores, ws, ws_bytes, stream, full != 0, row_lo, row_hi);
}

cc_status cc_partition_rows(const cc_model_cfg *cfg, int32_t full, const int32_t *seq_len,
                            int32_t batch, int32_t world, int32_t align, int32_t *row_lo,
                            int32_t *row_hi) {
  if (!cfg || !seq_len || !row_lo || !row_hi || batch < 1 || world < 1 || align < 1)
    return CC_ERR_INVALID_ARG;
  // the cost model needs positive sizes only (no kernel runs here)
  if (cfg->d_model < 1 || cfg->n_q_heads < 1 || cfg->head_dim < 1 || cfg->d_ff < 1)
    return CC_ERR_INVALID_ARG;
  (void)full;   // every layer repeats the same per-row work: the split is the same
  // per row and layer: projections 2 d (2 Hq dh) + 6 d F FLOPs, attention
  // 4 dh Hq per later slot
  const double g = 4.0 * cfg->d_model * (double)cfg->n_q_heads * cfg->head_dim +
                   6.0 * cfg->d_model * (double)cfg->d_ff;
  const double a = 4.0 * cfg->head_dim * (double)cfg->n_q_heads;
  for (int b = 0; b < batch; ++b) {
    const int64_t n = seq_len[b];
    if (n < 0) return CC_ERR_INVALID_ARG;
    // cost of rows [0, k): g k + a (k (n - 1) - k (k - 1) / 2), increasing in k
    auto cost = [&](int64_t k) {
      return g * k + a * ((double)k * (n - 1) - (double)k * (k - 1) / 2.0);
    };
    const double total = cost(n);
    int64_t prev = 0;
    for (int r = 0; r < world; ++r) {
      int64_t hi = n;
      if (r + 1 < world) {
        const double target = total * (r + 1) / world;
        int64_t lo_k = prev, hi_k = n;   // smallest k with cost(k) >= target
        while (lo_k < hi_k) {
          const int64_t mid = (lo_k + hi_k) / 2;
          if (cost(mid) >= target) hi_k = mid; else lo_k = mid + 1;
        }
        hi = std::min<int64_t>(n, std::max<int64_t>(prev, (lo_k + align / 2) / align * align));
      }
      row_lo[(size_t)r * batch + b] = (int32_t)prev;
      row_hi[(size_t)r * batch + b] = (int32_t)hi;
      prev = hi;
    }
  }
  return CC_OK;
}

size_t cc_select_workspace_size(int32_t batch, int32_t cap) {
  (void)batch;
  (void)cap;
  return 0;   // one CTA per sequence keeps its histograms in shared memory
}

cc_status cc_select_keep(const float *scores, const int32_t *seq_len, int32_t batch, int32_t cap,
                         const int32_t *budget, int32_t n_sink, int32_t *keep_idx,
                         int32_t *keep_count, void *ws, size_t ws_bytes, void *stream) {
  (void)ws;
  (void)ws_bytes;
  if (!scores || !seq_len || !budget || !keep_idx || !keep_count || batch < 1 || cap < 1 ||
      n_sink < 0)
    return CC_ERR_INVALID_ARG;
  DevState *dev;
  if (!dev_state(&dev)) return device_fail();
  TimedScope t(CC_KERNEL_SELECT, reinterpret_cast<cudaStream_t>(stream));
  CC_TRY(launch_select(scores, seq_len, batch, cap, budget, n_sink, keep_idx, keep_count,
                       dev->status, reinterpret_cast<cudaStream_t>(stream)));
  return CC_OK;
}

size_t cc_compact_workspace_size(const cc_model_cfg *cfg, const cc_kv_cache *cache) {
  CompactPlan plan;
  if (compact_plan(cfg, cache, plan) != CC_OK) return 0;
  return plan.ws_bytes;
}

cc_status cc_compact_kv(const cc_model_cfg *cfg, const cc_kv_cache *cache,
                        const int32_t *keep_idx, const int32_t *keep_count, void *ws,
                        size_t ws_bytes, void *stream) {
  static CompactPlan plan;   // large (kernel parameter block); guarded below
  static std::mutex mu;
  std::lock_guard<std::mutex> lk(mu);
  cc_status s = compact_plan(cfg, cache, plan);
  if (s != CC_OK) return s;
  if (!keep_idx || !keep_count) return CC_ERR_INVALID_ARG;
  if (!ws || !aligned16(ws) || ws_bytes < plan.ws_bytes) return CC_ERR_WORKSPACE;
  DevState *dev;
  if (!dev_state(&dev)) return device_fail();
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if ((s = compact_bind(plan, ws, st)) != CC_OK) return s;
  plan.p.keep_idx = keep_idx;
  plan.p.keep_count = keep_count;
  plan.p.seq_len = cache->seq_len;
  plan.p.status = dev->status;
  plan.p.withhold_unit = g_withhold_unit;
  g_withhold_unit = -1;
  CC_TRY(wait_kv_ready(cache, 0, cfg->n_layers, st));
  TimedScope t(CC_KERNEL_COMPACT, st);
  CC_TRY(launch_compact(plan.p, dev->sms, st));
  return CC_OK;
}

cc_status cc_get_status(void *stream) {
  DevState *dev;
  if (!dev_state(&dev)) return device_fail();
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(st) != cudaSuccess) return CC_ERR_CUDA;
  unsigned v = 0;
  if (cudaMemcpy(&v, dev->status, sizeof(v), cudaMemcpyDeviceToHost) != cudaSuccess)
    return CC_ERR_CUDA;
  const unsigned zero = 0;
  if (cudaMemcpy(dev->status, &zero, sizeof(zero), cudaMemcpyHostToDevice) != cudaSuccess)
    return CC_ERR_CUDA;
  return static_cast<cc_status>(v);
}

const char *cc_last_error(void) { return g_last_error; }

const char *cc_status_str(cc_status s) {
  switch (s) {
    case CC_OK: return "ok";
    case CC_ERR_INVALID_ARG: return "invalid argument";
    case CC_ERR_CUDA: return "CUDA error";
    case CC_ERR_BUDGET: return "budget below the forced keeps";
    case CC_ERR_WORKSPACE: return "workspace too small";
    case CC_ERR_TIMEOUT: return "device wait timed out";
    case CC_ERR_UNSUPPORTED: return "unsupported shape";
    case CC_ERR_DEVICE_ARG: return "device-side argument out of range";
    case CC_ERR_RANGE: return "value outside the fp16 range";
  }
  return "unknown status";
}

// ---- kernel-level entry points (include/cc_kernels.h) ----------------------

cc_status cc_linear_f32(const void *x, const void *w, float *y, int32_t rows, int32_t n,
                        int32_t k, void *stream) {
  if (!x || !w || !y || rows < 1 || n < 1 || k < 1 || n % 32 || k % 8) return CC_ERR_INVALID_ARG;
  if (!aligned16(x) || !aligned16(w) || !aligned16(y)) return CC_ERR_INVALID_ARG;
  DevState *dev;
  if (!dev_state(&dev)) return device_fail();
  Gemm g;
  cc_status s = gemm_setup(g, EPI_F32, x, k, w, nullptr, n, 1, rows, nullptr, dev->status);
  if (s != CC_OK) return s;
  g.p.out = y;
  g.p.ldo = n;
  return run_gemm(g, EPI_F32, CC_KERNEL_OTHER, dev->sms, reinterpret_cast<cudaStream_t>(stream));
}

static cc_status attention_entry(const void *q, const void *k, const void *v,
                                 const int32_t *seq_len, void *out, int32_t batch, int32_t cap,
                                 int32_t n_q_heads, int32_t n_kv_heads, int32_t head_dim,
                                 void *stream, bool split) {
  if (!q || !k || !v || !seq_len || !out || batch < 1 || cap < 1 || n_q_heads < 1 ||
      n_kv_heads < 1 || n_q_heads % n_kv_heads)
    return CC_ERR_INVALID_ARG;
  if (head_dim != 64 && head_dim != 128) return CC_ERR_UNSUPPORTED;
  if (n_q_heads / n_kv_heads > 256) return CC_ERR_UNSUPPORTED;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(out)) return CC_ERR_INVALID_ARG;
  if ((uint64_t)batch * cap >= (1ull << 31)) return CC_ERR_UNSUPPORTED;
  DevState *dev;
  if (!dev_state(&dev)) return device_fail();
  cc_model_cfg c{};
  c.n_q_heads = n_q_heads;
  c.n_kv_heads = n_kv_heads;
  c.head_dim = head_dim;
  return run_attention(&c, q, k, v, out, seq_len, batch, cap, dev->status,
                       reinterpret_cast<cudaStream_t>(stream), split, nullptr, 0, nullptr, 0,
                       KvFmt(), split);
}

cc_status cc_counter_causal_attention(const void *q, const void *k, const void *v,
                                      const int32_t *seq_len, void *out, int32_t batch,
                                      int32_t cap, int32_t n_q_heads, int32_t n_kv_heads,
                                      int32_t head_dim, void *stream) {
  return attention_entry(q, k, v, seq_len, out, batch, cap, n_q_heads, n_kv_heads, head_dim,
                         stream, false);
}

cc_status cc_counter_causal_attention_split(const void *q, const void *k, const void *v,
                                            const int32_t *seq_len, void *out, int32_t batch,
                                            int32_t cap, int32_t n_q_heads, int32_t n_kv_heads,
                                            int32_t head_dim, void *stream) {
  return attention_entry(q, k, v, seq_len, out, batch, cap, n_q_heads, n_kv_heads, head_dim,
                         stream, true);
}

// ---- captured call sequences ------------------------------------------------

struct cc_graph {
  cudaGraphExec_t exec;
};

cc_status cc_graph_begin(void *stream) {
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (!st) return CC_ERR_INVALID_ARG;   // the legacy default stream cannot be captured
  {
    std::lock_guard<std::mutex> lk(g_mu);
    if (g_timing.on) return CC_ERR_INVALID_ARG;
  }
  DevState *dev;
  if (!dev_state(&dev)) return device_fail();
  CC_TRY(cudaStreamBeginCapture(st, cudaStreamCaptureModeThreadLocal));
  return CC_OK;
}

cc_status cc_graph_end(void *stream, cc_graph **out) {
  if (out) *out = nullptr;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (!st) return CC_ERR_INVALID_ARG;
  cudaGraph_t graph = nullptr;
  cudaError_t e = cudaStreamEndCapture(st, &graph);
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamEndCapture");
  if (!out) {
    cudaGraphDestroy(graph);
    return CC_ERR_INVALID_ARG;
  }
  cudaGraphExec_t exec = nullptr;
  e = cudaGraphInstantiate(&exec, graph, 0);
  cudaGraphDestroy(graph);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGraphInstantiate");
  *out = new cc_graph{exec};
  return CC_OK;
}

cc_status cc_graph_launch(const cc_graph *g, void *stream) {
  if (!g) return CC_ERR_INVALID_ARG;
  CC_TRY(cudaGraphLaunch(g->exec, reinterpret_cast<cudaStream_t>(stream)));
  return CC_OK;
}

cc_status cc_graph_destroy(cc_graph *g) {
  if (!g) return CC_OK;
  cudaError_t e = cudaGraphExecDestroy(g->exec);
  delete g;
  if (e != cudaSuccess) return cuda_fail(e, "cudaGraphExecDestroy");
  return CC_OK;
}

// ---- launch timing (include/cc_profile.h) ----------------------------------

cc_status cc_timing_enable(int32_t on) {
  std::lock_guard<std::mutex> lk(g_mu);
  for (auto &r : g_timing.recs) {
    g_timing.pool.push_back(r.a);
    g_timing.pool.push_back(r.b);
  }
  g_timing.recs.clear();
  g_timing.on = on != 0;
  return CC_OK;
}

cc_status cc_timing_collect(int32_t *counts, double *total_ms) {
  if (!counts || !total_ms) return CC_ERR_INVALID_ARG;
  std::lock_guard<std::mutex> lk(g_mu);
  for (int k = 0; k < CC_KERNEL_COUNT; ++k) {
    counts[k] = 0;
    total_ms[k] = 0.0;
  }
  cc_status st = CC_OK;
  for (auto &r : g_timing.recs) {
    float ms = 0.f;
    if (cudaEventSynchronize(r.b) != cudaSuccess || cudaEventElapsedTime(&ms, r.a, r.b) != cudaSuccess)
      st = CC_ERR_CUDA;
    if (r.kind >= 0 && r.kind < CC_KERNEL_COUNT) {
      counts[r.kind] += 1;
      total_ms[r.kind] += ms;
    }
    g_timing.pool.push_back(r.a);
    g_timing.pool.push_back(r.b);
  }
  g_timing.recs.clear();
  return st;
}

cc_status cc_debug_withhold_compact_unit(int32_t unit) {
  g_withhold_unit = unit;
  return CC_OK;
}

const char *cc_kernel_name(int32_t kind) {
  static const char *names[CC_KERNEL_COUNT] = {
      "rmsnorm", "embed", "gemm_qrope", "attention", "gemm_oproj", "gemm_gateup", "gemm_down",
      "head_logit", "gemm_lmhead", "lse_combine", "select", "compact", "other",
      "gemm_kv", "attention_causal", "append", "gemm_qkv", "keyattn", "kv_dequant"};
  return (kind >= 0 && kind < CC_KERNEL_COUNT) ? names[kind] : "unknown";
}

}  // extern "C"

// ---- library-internal helpers (internal.h) ----------------------------------
#include "internal.h"

namespace cc {

// cc_kv_cache.kv_ready: the caller's uploads of layers [l0, l1) land before what follows on st
cudaError_t wait_kv_ready(const cc_kv_cache *kv, int l0, int l1, cudaStream_t st) {
  if (!kv->kv_ready) return cudaSuccess;
  for (int l = l0; l < l1; ++l) {
    if (!kv->kv_ready[l]) continue;
    const cudaError_t e = cudaStreamWaitEvent(st, reinterpret_cast<cudaEvent_t>(kv->kv_ready[l]), 0);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}


cc_status compact_plan_bind(const cc_model_cfg *cfg, const cc_kv_cache *cache, CompactParams &p,
                            void *scratch, size_t scratch_cap, cudaStream_t st) {
  static CompactPlan plan;
  static std::mutex mu;
  std::lock_guard<std::mutex> lk(mu);
  cc_status s = compact_plan(cfg, cache, plan);
  if (s != CC_OK) return s;
  if (plan.ws_bytes > scratch_cap) return CC_ERR_WORKSPACE;
  if ((s = compact_bind(plan, scratch, st)) != CC_OK) return s;
  p = plan.p;
  return CC_OK;
}

cudaError_t launch_compact_timed(const CompactParams &p, int sms, cudaStream_t st) {
  TimedScope t(CC_KERNEL_COMPACT, st);
  return launch_compact(p, sms, st);
}

bool current_device_info(unsigned **status, int *sms) {
  DevState *d;
  if (!dev_state(&d)) return false;
  *status = d->status;
  *sms = d->sms;
  return true;
}

}  // namespace cc
