/*
 * cc_profile.h -- optional launch timing of the counter-causal refresh
 * library.  When enabled, every kernel the library launches is bracketed by
 * two CUDA events recorded on the launch's own stream; cc_timing_collect
 * waits for the recorded events and returns, per kernel kind, the number of
 * launches and their summed duration.  Used by benchmarks to attribute a
 * refresh's time to its kernels; off by default.  Not thread-safe against
 * concurrent library calls from several host threads while enabled.
 */
#ifndef CC_PROFILE_H_
#define CC_PROFILE_H_

#include "cc.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  CC_KERNEL_RMSNORM = 0,     /* RMSNorm rows -> bf16                              */
  CC_KERNEL_EMBED = 1,       /* embedding gather (full pass)                      */
  CC_KERNEL_GEMM_QROPE = 2,  /* query projection + RoPE                           */
  CC_KERNEL_ATTENTION = 3,   /* counter-causal attention                          */
  CC_KERNEL_GEMM_OPROJ = 4,  /* output projection + residual                      */
  CC_KERNEL_GEMM_GATEUP = 5, /* gate/up projection + SwiGLU                       */
  CC_KERNEL_GEMM_DOWN = 6,   /* down projection + residual                        */
  CC_KERNEL_HEAD_LOGIT = 7,  /* final norm + target-logit gather-dot              */
  CC_KERNEL_GEMM_LMHEAD = 8, /* LM-head GEMM + log-sum-exp partials (log-prob)    */
  CC_KERNEL_LSE_COMBINE = 9, /* log-sum-exp combine (log-prob)                    */
  CC_KERNEL_SELECT = 10,     /* keep-set radix select                             */
  CC_KERNEL_COMPACT = 11,    /* in-place compaction                               */
  CC_KERNEL_OTHER = 12,      /* kernel-level entry points (cc_kernels.h)          */
  CC_KERNEL_GEMM_KV = 13,    /* key (+ RoPE) and value projections (append)       */
  CC_KERNEL_ATTN_CAUSAL = 14,/* memory-augmented causal attention (append)        */
  CC_KERNEL_APPEND = 15,     /* append bookkeeping: tokens, positions, H^(L-1)    */
  CC_KERNEL_GEMM_QKV = 16,   /* fused q/k/v projections (+ RoPE) of the append    */
  CC_KERNEL_KEYATTN = 17,    /* comparison scorers: attention received per key    */
  CC_KERNEL_KV_DEQUANT = 18, /* a layer's K/V copied for the tile attention: e4m3
                                as bf16 or fp16, bf16 as fp16 (CC_SCORE_F16)        */
  CC_KERNEL_COUNT = 19
} cc_kernel_kind;

/* on != 0: start recording (also clears earlier records); 0: stop. */
cc_status cc_timing_enable(int32_t on);
/* Synchronises the recorded events; writes counts[k] launches and
 * total_ms[k] summed milliseconds for k < CC_KERNEL_COUNT (host arrays),
 * then clears the records. */
cc_status cc_timing_collect(int32_t *counts, double *total_ms);
const char *cc_kernel_name(int32_t kind);

/* Failure-path test hook.  The next cc_compact_kv call (only that one) runs
 * with work unit `unit` (units numbered array by array, K_0, V_0, K_1, ...,
 * then H, tokens, positions; in each, the kept-slot chunks in ascending
 * order) never publishing its "sources read"
 * flag, as if that unit had stalled: a unit that depends on it waits out its
 * bounded wait (about 2 s), skips its writes and records CC_ERR_TIMEOUT, and
 * the kernel returns normally.  The GPU context stays usable.  -1 disarms. */
cc_status cc_debug_withhold_compact_unit(int32_t unit);

#ifdef __cplusplus
}
#endif
#endif /* CC_PROFILE_H_ */
