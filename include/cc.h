/*
 * cc.h -- C ABI of the counter-causal KV-cache refresh (arXiv 2607.27600).
 *
 * One memory refresh (Algorithm DoMemRefresh) is three calls on one CUDA
 * stream:
 *   1. cc_score_layer / cc_score_full: the counter-causal surprise score of
 *      every cached slot (Sec. 3.1, Eq. 5 and the logit score it uses);
 *   2. cc_select_keep: the keep-set, the J highest scores (argsort, keep
 *      sigma[1:J]);
 *   3. cc_compact_kv: K' <- (K' (+) K)_sigma[1:J], V', X likewise, in place.
 *
 * Conventions for every call:
 *   - The caller owns all memory.  Every tensor argument is a device pointer
 *     unless documented as host.  The library allocates nothing; scratch
 *     lives in a caller-provided device workspace `ws` of at least the size
 *     the matching *_workspace_size call returns (256-byte aligned).
 *   - Calls are asynchronous on `stream` (a cudaStream_t; NULL = legacy
 *     default stream).  Errors found on the host (null or misaligned
 *     pointers, bad sizes, workspace too small, unsupported shapes) are
 *     returned at once and nothing is enqueued.  Errors found on the device
 *     (seq_len outside [0, cap], a budget below the forced keeps, an
 *     internal wait that timed out) are recorded in a per-device status word
 *     that cc_get_status reads and clears; the offending kernel skips the
 *     affected work instead of faulting.
 *   - bf16 means IEEE bfloat16 (2 bytes).  Matrices are row-major.  Weight
 *     matrices use the nn.Linear layout [out_features][in_features].
 *   - Row-major device buffers must start on a 16-byte boundary and have
 *     rows whose byte size is a multiple of 16.
 */
#ifndef CC_H_
#define CC_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  CC_OK = 0,
  CC_ERR_INVALID_ARG = 1,  /* null/misaligned pointer, bad size or shape          */
  CC_ERR_CUDA = 2,         /* a CUDA runtime call failed                           */
  CC_ERR_BUDGET = 3,       /* device: budget < forced keeps (1 + n_sink)           */
  CC_ERR_WORKSPACE = 4,    /* workspace smaller than *_workspace_size              */
  CC_ERR_TIMEOUT = 5,      /* device: an internal wait gave up (kernel returned)   */
  CC_ERR_UNSUPPORTED = 6,  /* shape outside what the kernels implement             */
  CC_ERR_DEVICE_ARG = 7,   /* device: seq_len/keep_count outside [0, cap]          */
  CC_ERR_RANGE = 8         /* device: a value written as an fp16 operand (mode
                              CC_SCORE_F16, cc_bf16_to_f16) exceeded 65504         */
} cc_status;

/* Score definition.  Sec. 3.1 takes the logit of the row's own token x_i as
 * the score; Eq. 5 defines surprise as 1 - P(x_i | x_{i+1:t}).  Both are
 * returned with the sign that makes "more surprising" rank higher. */
typedef enum {
  CC_SCORE_LOGIT = 0,   /* score_i = -z_i[x_i], z_i = final-norm(h_i) W_U^T      */
  CC_SCORE_LOGPROB = 1, /* score_i = -log softmax(z_i)[x_i] (same order as Eq. 5) */
  /* Flag, OR-ed into the mode, either pass: carry every tensor-core operand
   * that is not an exact bf16 input -- the GEMM activations (normalised
   * inputs, attention output, SwiGLU output), the queries entering Q K^T and
   * the attention probabilities entering P V -- as a bf16 pair hi + lo
   * (hi = bf16(x), lo = bf16(x - hi): ~2^-17 relative) instead of one bf16
   * value; each product then runs once per half (about twice the cost of the
   * pass).  Weights, cached K/V and H^(L-1) are bf16 inputs and stay exact.
   * Without it a deep random-weight model drifts from the exact score over
   * depth by several percent; with it the 32-layer score stays within
   * ~1e-3.  An e4m3 cache's codes enter the attention as exact bf16
   * values (the scales applied in fp32), so the same holds. */
  CC_SCORE_PRECISE = 0x100,
  /* Flag, OR-ed into the mode of cc_score_rows: the rows of the range are
   * written and every other entry of scores (other rows, slots past the
   * sequence ends) keeps its value, so that calls over disjoint ranges fill
   * one buffer -- e.g. blocks of rows scored as their inputs arrive. */
  CC_SCORE_RANGE_ONLY = 0x200,
  /* Flag, OR-ed into the mode, either pass (not with CC_SCORE_PRECISE): every
   * tensor-core operand of the layers in fp16 instead of bf16 -- one value,
   * not a pair, so the pass costs what the default one does.  fp16 keeps 11
   * significant bits to bf16's 8, so each rounding is 8x smaller, and it
   * represents every bf16 value of magnitude in [2^-14, 65504] exactly:
   *   - wq, wo, w_gate, w_up and w_down of layers[] are fp16 here (same
   *     shapes; cc_bf16_to_f16 converts the bf16 weights once);
   *   - the cached K/V (bf16 or e4m3) are copied to fp16 per layer in the
   *     workspace's activation buffer (needs 4 * Hkv * head_dim <= 2 * d_ff
   *     bytes per slot, else CC_ERR_UNSUPPORTED);
   *   - the queries, the attention probabilities and the GEMM activations
   *     (normalised inputs, attention output, SwiGLU output) are written as
   *     fp16; a finite value above 65504 in magnitude is reported on the
   *     device as CC_ERR_RANGE (use the bf16 modes for such a model);
   *   - the gains, biases, embedding, lm_head, H^(L-1) and the head (final
   *     norm, logit or log-prob) stay as in the default mode.
   * On a deep random-weight model the 32-layer score stays within ~2e-2 of
   * the exact one, where single bf16 operands drift by several percent. */
  CC_SCORE_F16 = 0x400
} cc_score_mode;

/* Element format of the cached keys and values.  The paper keeps the model's
 * own precision; the e4m3 format is a variant that halves the cache: an
 * element is code * scale, with one scale per layer for K and one for V (the
 * OCP FP8 E4M3 code: bias 7, no infinities, largest finite 448).  The
 * scoring passes, the compaction, cc_append_chunk and cc_decode_step take
 * either format (appends write codes rounded to nearest, saturating at
 * +-448); the attention-based comparison scorers and
 * cc_counter_causal_attention take bf16 only (CC_ERR_UNSUPPORTED).  The
 * scoring passes and the append attend over an exact bf16 copy of each
 * layer's codes, made in the workspace's activation buffer (which needs
 * 4 * Hkv * head_dim <= 2 * d_ff bytes per slot, else CC_ERR_UNSUPPORTED). */
typedef enum {
  CC_KV_BF16 = 0,
  CC_KV_E4M3 = 1
} cc_kv_format;

/* Order of the cached K/V buffers of a (not paged) cache: slot-major
 * [batch][cap][Hkv][head_dim] (one slot's heads together), or head-major
 * [batch][Hkv][cap][head_dim] (each KV head's slots together, as many model
 * runtimes keep their caches).  Every entry point takes either. */
typedef enum {
  CC_KV_SLOT_MAJOR = 0,
  CC_KV_HEAD_MAJOR = 1
} cc_kv_layout;

/* Decoder shape (Llama/Qwen pre-norm block: RMSNorm, GQA attention with
 * rotate-half RoPE, RMSNorm, SwiGLU MLP; final RMSNorm; untied LM head). */
typedef struct {
  int32_t n_layers;
  int32_t d_model;
  int32_t n_q_heads;
  int32_t n_kv_heads;   /* n_q_heads % n_kv_heads == 0; q head t reads KV head t / (Hq/Hkv) */
  int32_t head_dim;     /* 64 or 128                                                        */
  int32_t d_ff;
  int32_t vocab;
  float rope_theta;     /* inv_freq_k = theta^(-2k/head_dim), angles taken exactly mod 2pi  */
  float rms_eps;
  /* Optional Llama-3.1 RoPE frequency scaling (a property of that model, not
   * of the paper's method).  0 = off (a zero-initialised struct has it off).
   * Otherwise, with wavelength w_k = 2 pi / inv_freq_k: w_k below
   * original_max_pos / high_freq_factor keeps inv_freq_k; above
   * original_max_pos / low_freq_factor it becomes inv_freq_k / factor; in
   * between, (1 - a) inv_freq_k / factor + a inv_freq_k with
   * a = (original_max_pos / w_k - low) / (high - low).
   * Requires factor >= 1, 0 < low < high, original_max_pos > 0
   * (else CC_ERR_INVALID_ARG). */
  float rope_scaling_factor;
  float rope_low_freq_factor;
  float rope_high_freq_factor;
  int32_t rope_original_max_pos;
} cc_model_cfg;

/* One layer's weights, all bf16 device pointers. */
typedef struct {
  const void *attn_norm; /* [d_model]                        */
  const void *wq;        /* [n_q_heads*head_dim][d_model]    */
  const void *wo;        /* [d_model][n_q_heads*head_dim]    */
  const void *mlp_norm;  /* [d_model]                        */
  const void *w_gate;    /* [d_ff][d_model]                  */
  const void *w_up;      /* [d_ff][d_model]                  */
  const void *w_down;    /* [d_model][d_ff]                  */
  const void *bq;        /* optional [n_q_heads*head_dim] q-projection bias (Qwen2-style
                            attention), added before RoPE; NULL = none; 16-byte aligned   */
  /* Key/value projections, read only by cc_append_chunk (the scoring passes
   * reuse the cached K/V and may leave them NULL). */
  const void *wk;        /* [n_kv_heads*head_dim][d_model]   */
  const void *wv;        /* [n_kv_heads*head_dim][d_model]   */
  const void *bk;        /* optional [n_kv_heads*head_dim] bias (before RoPE); NULL = none */
  const void *bv;        /* optional [n_kv_heads*head_dim] bias; NULL = none              */
} cc_layer_weights;

typedef struct {
  const void *embed;                /* bf16 [vocab][d_model] (full pass only)       */
  const void *final_norm;           /* bf16 [d_model]                               */
  const void *lm_head;              /* bf16 [vocab][d_model]                        */
  const cc_layer_weights *layers;   /* HOST array [n_layers]; the fast pass reads
                                       only layers[n_layers-1]                      */
} cc_model_weights;

/* A batch of cached sequences in slot-major buffers of `cap` slots each.
 * Sequence b holds seq_len[b] valid slots [0, seq_len[b]); slots past that
 * are ignored (they may hold any bits).  K is stored post-RoPE (Sec. 3.1). */
typedef struct {
  int32_t batch;
  int32_t cap;
  int32_t *seq_len;  /* device int32 [batch]; cc_compact_kv sets it to keep_count     */
  void *const *k;    /* HOST array [n_layers] of device [batch][cap][Hkv][head_dim]
                        elements (bf16, or e4m3 bytes: kv_format); an entry may be
                        NULL where a call does not need that layer                     */
  void *const *v;    /* same layout as k                                               */
  int32_t *tokens;   /* device int32 [batch][cap]: the token buffer X                  */
  int32_t *pos;      /* device int32 [batch][cap]: original position ids (>= 0)        */
  void *h_last;      /* device bf16 [batch][cap][d_model]: H^(L-1), the input of the
                        last layer recorded by the causal pass (fast mode); may be NULL
                        for cc_score_full                                               */
  float *h2o_acc;    /* optional device fp32 [batch][cap]: running totals of the H2O
                        comparison scorer (cc_h2o_accumulate), compacted with the cache;
                        NULL when unused                                                */
  int32_t kv_format; /* cc_kv_format of k and v (0 = bf16)                               */
  const float *kv_scale; /* CC_KV_E4M3: HOST array [n_layers][2] = (K scale, V scale) of
                        each layer, finite and > 0; the value of an element is its code
                        times the scale.  Ignored for bf16.                             */
  /* Paged K/V (NULL block_table: k[l], v[l] are slot-major [batch][cap] buffers).
   * With a block table, k[l] and v[l] are page pools [n_pages][page_size][Hkv][head_dim]
   * and logical slot i of sequence b lives at pool row
   *   block_table[b * (cap / page_size) + i / page_size] * page_size + i % page_size.
   * page_size is a multiple of 128 and divides cap; every entry a sequence uses
   * (slots below cap) names a distinct page in [0, n_pages) (an entry outside that range
   * is reported as CC_ERR_DEVICE_ARG on the device and its rows are skipped).  Only K
   * and V are paged: tokens, pos, h_last and h2o_acc stay [batch][cap].  The compaction
   * moves rows between the pages of a sequence and leaves the table as it is: pages past
   * the new length are the caller's to reuse. */
  const int32_t *block_table; /* device int32 [batch][cap / page_size], or NULL          */
  int32_t page_size;
  int32_t n_pages;
  int32_t kv_layout;  /* cc_kv_layout of k and v (0 = slot-major); a head-major cache is
                         not paged                                                      */
  /* Optional HOST array [n_layers] of cudaEvent_t (as void *; the array or any entry may
   * be NULL): the caller's writes of layer l's K/V may still be in flight on another
   * stream when a call is enqueued; the call's stream waits for kv_ready[l] right before
   * its first kernel that reads or writes layer l's K/V (the scoring pass before layer
   * l's attention, the append and decode at the start of layer l, the comparison scorers
   * and the compaction before their launch), so an upload of the cache overlaps the
   * kernels that do not need it.  Leave kv_ready NULL for calls recorded into a graph
   * (cc_graph_begin): the waits are for eager calls whose inputs are still arriving. */
  void *const *kv_ready;
} cc_kv_cache;

/* ---- scoring (Sec. 3.1) ---------------------------------------------------
 * Writes scores[b*cap + i] (fp32, device [batch][cap]) for every slot
 * i < seq_len[b]; slot seq_len[b]-1 gets +inf (the last token has no future
 * context and is always retained); slots >= seq_len[b] get -inf.
 *
 * cc_score_layer -- fast single-layer approximation: queries from h_last
 * with RoPE at pos, counter-causal attention (row i attends slots j with
 * i < j < seq_len[b]) over k[n_layers-1], v[n_layers-1], then the rest of
 * the last layer, the final norm and the head.
 * cc_score_full -- full pass: embedding of tokens, every layer l with fresh
 * queries over k[l], v[l] (reused, not recomputed), final norm, head.
 */
/* Workspace bytes for either pass in `mode` (with CC_SCORE_PRECISE: the
 * layout with [hi | lo] activation rows). */
size_t cc_score_workspace_size(const cc_model_cfg *cfg, int32_t batch, int32_t cap,
                               cc_score_mode mode);
cc_status cc_score_layer(const cc_model_cfg *cfg, const cc_model_weights *w,
                         const cc_kv_cache *cache, cc_score_mode mode, float *scores,
                         void *ws, size_t ws_bytes, void *stream);
cc_status cc_score_full(const cc_model_cfg *cfg, const cc_model_weights *w,
                        const cc_kv_cache *cache, cc_score_mode mode, float *scores,
                        void *ws, size_t ws_bytes, void *stream);

/* cc_bf16_to_f16 -- dst[i] = fp16(src[i]) for i < n: the weight matrices of
 * mode CC_SCORE_F16, converted once before the scoring calls.  Exact for
 * magnitudes in [2^-14, 65504] (and zero); smaller ones round to the nearest
 * multiple of 2^-24 (ties to even); a larger finite value becomes +-inf and
 * is reported as CC_ERR_RANGE on the device (cc_get_status).  NaN and inf
 * pass through.  src, dst: device, 16-byte aligned, not overlapping; n a
 * multiple of 8 (else CC_ERR_INVALID_ARG); n = 0 does nothing.  Async on
 * `stream`. */
cc_status cc_bf16_to_f16(const void *src, void *dst, size_t n, void *stream);

/* ---- one refresh sharded over several GPUs by query rows ----------------------
 * Given the cache, a row's score depends only on its own input (token or
 * H^(L-1) row) and on the cached K/V of the later slots, which the pass
 * reuses without recomputing them (Sec. 3.1); so the rows of one refresh
 * can be split between processes that each hold the cache.
 *
 * cc_score_rows -- cc_score_layer (full = 0) or cc_score_full (full = 1)
 * restricted to the rows row_lo[b] <= i < row_hi[b] of each sequence
 * (row_lo, row_hi: device int32 [batch], 0 <= row_lo[b] <= row_hi[b] <=
 * seq_len[b], else CC_ERR_DEVICE_ARG on the device and those rows skipped).
 * Each row still attends every later slot up to seq_len[b].  Those rows get
 * their scores (slot seq_len[b]-1 gets +inf when in range) and every other
 * entry of scores [batch][cap] gets -inf, so the element-wise maximum of the
 * ranks' buffers (one MAX all-reduce of batch * cap floats) is the whole
 * refresh's scores; with CC_SCORE_RANGE_ONLY in mode the other entries are
 * left as they are instead.  A row's score is bit-identical to the one
 * cc_score_layer / cc_score_full writes for it with the same cache and mode.
 * Same workspace as those calls.  row_lo and row_hi must both be null (every
 * row) or both be given. */
cc_status cc_score_rows(const cc_model_cfg *cfg, const cc_model_weights *w,
                        const cc_kv_cache *cache, cc_score_mode mode, int32_t full,
                        const int32_t *row_lo, const int32_t *row_hi, float *scores, void *ws,
                        size_t ws_bytes, void *stream);

/* cc_partition_rows -- host-side plan: splits every sequence's rows [0,
 * seq_len[b]) into `world` contiguous blocks, block r for rank r, of equal
 * estimated cost.  A row's cost per layer is its projections' FLOPs (the
 * same for every row) plus its attention's, which grows with the number of
 * later slots, so the early rows cost more and get the shorter blocks.
 * Interior boundaries are multiples of `align` (>= 1; 128 matches the row
 * tiles of the projections).  seq_len: HOST int32 [batch]; row_lo, row_hi:
 * HOST int32 [world][batch] written with rank r's block of sequence b at
 * [r * batch + b].  The blocks of a sequence are disjoint, ascending and
 * cover it exactly (a short sequence leaves some blocks empty).  Needs no
 * GPU.  CC_ERR_INVALID_ARG on null pointers, world < 1, align < 1 or a
 * negative length. */
cc_status cc_partition_rows(const cc_model_cfg *cfg, int32_t full, const int32_t *seq_len,
                            int32_t batch, int32_t world, int32_t align, int32_t *row_lo,
                            int32_t *row_hi);

/* ---- keep-set (Algorithm DoMemRefresh: sigma = argsort, keep sigma[1:J]) ---
 * For each sequence b keeps J_b = min(budget[b], seq_len[b]) slots: the
 * highest scores, ties broken toward the later slot, NaN ranked as -inf,
 * slots [0, n_sink) forced (frozen system-prompt slots, Sec. 3.2).
 * Writes keep_idx[b*cap + k], k < J_b, in ascending slot order, and
 * keep_count[b] = J_b.  Entries of keep_idx past J_b are not written.
 * scores, seq_len, budget: device; keep_idx [batch][cap], keep_count [batch]:
 * device.  A budget below min(seq_len, 1 + n_sink) sets CC_ERR_BUDGET on the
 * device and keeps the forced slots plus the last slot. */
size_t cc_select_workspace_size(int32_t batch, int32_t cap);
cc_status cc_select_keep(const float *scores, const int32_t *seq_len, int32_t batch,
                         int32_t cap, const int32_t *budget, int32_t n_sink,
                         int32_t *keep_idx, int32_t *keep_count, void *ws, size_t ws_bytes,
                         void *stream);

/* ---- compaction (Algorithm DoMemRefresh: K' <- (K' (+) K)_sigma[1:J]) ------
 * In place, for every sequence b and k < keep_count[b]: slot k of every
 * non-NULL k[l], v[l] (l < cfg->n_layers), of tokens, pos and (if non-NULL)
 * h_last receives old slot keep_idx[b*cap + k].  keep_idx must be strictly
 * ascending per sequence (as cc_select_keep writes it).  Slots >=
 * keep_count[b] keep their old contents.  Then seq_len[b] = keep_count[b]. */
size_t cc_compact_workspace_size(const cc_model_cfg *cfg, const cc_kv_cache *cache);
cc_status cc_compact_kv(const cc_model_cfg *cfg, const cc_kv_cache *cache,
                        const int32_t *keep_idx, const int32_t *keep_count, void *ws,
                        size_t ws_bytes, void *stream);

/* ---- inference cycle, pre-fill (Algorithm CacheManagedInference with
 * DoInference over a chunk of tokens in batch, chunked refresh mode) -------
 * Appends count[b] tokens to sequence b after its seq_len[b] cached slots:
 * the chunk runs through every layer l with queries, keys and values from
 * its own hidden states (keys and queries rotated at the chunk's positions),
 * writes its keys and values into k[l], v[l] at slots [seq_len[b],
 * seq_len[b] + count[b]) (K <- K (+) k_t, V <- V (+) v_t), and attends every
 * cached memory slot plus the chunk causally (memory-augmented attention,
 * Eq. 3, causal mask: the chunk's slot i sees slots j <= i).  The chunk's
 * tokens (X <- X (+) x_t) and positions are written to tokens and pos, the
 * input of the last layer to h_last (if non-NULL, for the fast
 * approximation), and seq_len[b] grows by count[b].  No next token is
 * sampled (pre-fill).
 *   tokens_in: device int32 [batch][max_count], row b holds count[b] ids.
 *   pos_in:    device int32 [batch][max_count] original positions, or NULL:
 *              the positions following pos[b][seq_len[b]-1] (0 when empty).
 *   count:     device int32 [batch]; a count outside [0, max_count] or past
 *              cap sets CC_ERR_DEVICE_ARG on the device and appends nothing
 *              to that sequence.  NULL with max_count == 1: one token each.
 * Needs embed and, for every layer, wq, wk, wv, wo, the norms and the MLP
 * (biases optional); every k[l], v[l] non-NULL.  Asynchronous on `stream`;
 * the workspace is that of cc_append_workspace_size. */
size_t cc_append_workspace_size(const cc_model_cfg *cfg, int32_t batch, int32_t cap);
/* ---- inference cycle, decode (Algorithm CacheManagedInference, decode
 * phase; DoInference for one token with greedy sampling, as in the paper's
 * experiments) ----------------------------------------------------------------
 * Appends tokens_in[b] (device int32 [batch], the current token x_t of each
 * sequence) exactly as cc_append_chunk with one token each, then applies the
 * final norm and the LM head to that position and writes the next token
 * next_tokens[b] = argmax of the logits (the lowest id on ties; -1 for a
 * sequence that could not append: full cache, reported on the device) and,
 * if next_logit is non-NULL, its logit.  Needs everything cc_append_chunk
 * needs plus final_norm and lm_head.  Each sequence's row is its own GEMM row
 * tile: one sequence reads the weights once per step, a batch of B reads
 * them B times (decode batching across sequences is not fused). */
size_t cc_decode_workspace_size(const cc_model_cfg *cfg, int32_t batch, int32_t cap);
cc_status cc_decode_step(const cc_model_cfg *cfg, const cc_model_weights *w,
                         const cc_kv_cache *cache, const int32_t *tokens_in,
                         int32_t *next_tokens, float *next_logit, void *ws, size_t ws_bytes,
                         void *stream);
cc_status cc_append_chunk(const cc_model_cfg *cfg, const cc_model_weights *w,
                          const cc_kv_cache *cache, const int32_t *tokens_in,
                          const int32_t *pos_in, const int32_t *count, int32_t max_count,
                          void *ws, size_t ws_bytes, void *stream);

/* ---- the paper's comparison scorers (Sec. 4) -------------------------------
 * They rank the same cached slots for the same cc_select_keep and
 * cc_compact_kv; the attention-based ones read only the cached keys, which
 * act as proxy queries (query slot i attends slots j <= i, softmax of
 * K[i] . K[j] / sqrt(head_dim) per KV head).  scores: device fp32
 * [batch][cap], -inf past seq_len.
 *
 * cc_score_recency -- sliding window (first in, first out): score = the
 *   slot's original position, so the keep-set is the most recent slots.
 * cc_score_importance -- importance: mean attention a slot receives in the
 *   last layer, over the KV heads and the n - j proxy queries that see it.
 * cc_h2o_accumulate -- heavy hitter (H2O): adds to cache->h2o_acc the
 *   attention each slot receives from the `recent` most recent keys as proxy
 *   queries, summed over KV heads and every layer (a running total across
 *   refreshes; zero it once when the cache starts).
 * cc_score_h2o -- H2O refresh scores: h2o_acc, with the `recent` most recent
 *   slots always kept (+inf).
 * The attention-based scorers need head_dim 64 or 128 and the workspace of
 * cc_keyattn_workspace_size; results are deterministic (fixed summation
 * order). */
cc_status cc_score_recency(const cc_kv_cache *cache, float *scores, void *stream);
size_t cc_keyattn_workspace_size(const cc_model_cfg *cfg, int32_t batch, int32_t cap);
cc_status cc_score_importance(const cc_model_cfg *cfg, const cc_kv_cache *cache, float *scores,
                              void *ws, size_t ws_bytes, void *stream);
cc_status cc_h2o_accumulate(const cc_model_cfg *cfg, const cc_kv_cache *cache, int32_t recent,
                            void *ws, size_t ws_bytes, void *stream);
cc_status cc_score_h2o(const cc_kv_cache *cache, int32_t recent, float *scores, void *stream);

/* ---- compaction without a workspace -----------------------------------------
 * The paper has no counterpart: this is a library convenience.
 * Same operation, checks and results as cc_compact_kv, for callers that
 * cannot allocate device memory for a workspace when they compact -- for
 * example a serving loop that has handed the whole device pool to the KV
 * cache, or a runtime that forbids device allocation on its refresh path
 * (cudaMalloc may block and synchronise the device).  Its scratch (a table
 * of work units, one flag per work unit and a table of which work units
 * read each destination chunk) lives in a fixed 1 MiB array in the
 * library's device memory, which every GPU that loads the library holds
 * until the process exits.  The call allocates nothing.
 *   - A cache needing more than 1 MiB of scratch (cc_compact_workspace_size()
 *     above 1 MiB) is rejected with CC_ERR_WORKSPACE before anything is
 *     enqueued.
 *   - The first call on a device looks up the array's device address (with
 *     that device current); make that first call before any stream capture.
 *   - All calls on a device share the array and each call clears it first
 *     (an asynchronous memset on `stream`): calls whose work overlaps on the
 *     GPU (different streams, no ordering between them) race on it and must
 *     not be issued. */
cc_status cc_compact_kv_static(const cc_model_cfg *cfg, const cc_kv_cache *cache,
                               const int32_t *keep_idx, const int32_t *keep_count,
                               void *stream);

/* ---- captured call sequences (CUDA graphs) -----------------------------------
 * The paper has no counterpart: this is a library convenience for
 * launch-bound loops (a decode step launches several kernels per layer for
 * one row each, so the host's launch latency, not the GPU, sets its pace).
 * cc_graph_begin starts capturing `stream` (a stream the caller created: the
 * legacy default stream cannot be captured; the capture is local to the
 * calling host thread); the cc_* calls that follow on that stream and thread
 * enqueue nothing but are recorded; cc_graph_end stops the capture and
 * returns an executable graph in *out, which cc_graph_launch replays on any
 * stream as one launch.
 *   - A replay repeats the recorded calls with the same arguments: the same
 *     pointers, sizes and host values.  What the kernels read from device
 *     memory (seq_len, counts, tokens, positions, keep-sets) is read afresh
 *     at each replay, so a captured decode step or refresh cycle replays over
 *     a cache that has grown or been compacted since.
 *   - Make each call once without capture first (first calls on a device
 *     set kernel attributes and look up device addresses), and keep launch
 *     timing (cc_timing_enable) off while capturing: cc_graph_begin returns
 *     CC_ERR_INVALID_ARG otherwise.
 *   - A captured call that returns an error leaves a partial recording:
 *     still call cc_graph_end (the stream leaves capture mode), then destroy
 *     what it returns.
 *   - cc_graph_end returns CC_ERR_CUDA (and *out = NULL) when the capture
 *     was invalidated or the graph cannot be instantiated. */
typedef struct cc_graph cc_graph;
cc_status cc_graph_begin(void *stream);
cc_status cc_graph_end(void *stream, cc_graph **out);
cc_status cc_graph_launch(const cc_graph *g, void *stream);
cc_status cc_graph_destroy(cc_graph *g);

/* ---- status ---------------------------------------------------------------
 * Synchronises `stream`, returns the first device-side error recorded since
 * the last call (CC_OK if none) on the current device and clears it.
 * Returns CC_ERR_CUDA if the stream itself reports a CUDA error. */
cc_status cc_get_status(void *stream);
const char *cc_status_str(cc_status s);
/* Text of the last CUDA error behind a CC_ERR_CUDA returned on this host
 * thread (the failing call and the CUDA error name); "" if none. */
const char *cc_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* CC_H_ */
