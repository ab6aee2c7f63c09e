// select.cu -- keep-set selection (Algorithm DoMemRefresh: sigma = argsort of
// the surprise scores, largest first; keep sigma[1:J]).
//
// One CTA (1024 threads) per sequence.  Each slot j gets the unique 64-bit
// key (monotone(score_j) << 32) | j, so "descending score, ties toward the
// later slot" is plain descending key order and exactly J keys are >= the
// J-th largest key T.  T is found by an MSB radix select (8 bits per pass,
// warp-level digit search over a shared histogram, at most 8 passes); it
// stops early once the bucket holding the boundary has exactly as many keys
// as are still needed: then every key of the bucket is kept, and the prefix
// with all lower bits zero is a threshold with exactly J keys at or above it.
// A final pass flags key >= T and writes the kept slots in ascending slot
// order through a block-wide prefix scan.
#include "select.cuh"

namespace cc {

namespace {

constexpr int kThreads = 1024;
constexpr uint32_t kKeyPosInf = 0xFF800000u;   // monotone key of +inf
constexpr uint32_t kKeyNegInf = 0x007FFFFFu;   // monotone key of -inf

// float -> uint32 whose unsigned order is the float order; NaN ranks as -inf.
// -0.0 and +0.0 compare equal as floats, so both take the key of +0.0 (a
// score -logit is -0.0 for a logit of exactly zero); their tie then goes to
// the later slot like any other.
CC_DEV uint32_t monotone_key(float f) {
  uint32_t u = __float_as_uint(f);
  if ((u & 0x7F800000u) == 0x7F800000u && (u & 0x007FFFFFu)) return kKeyNegInf;
  if ((u & 0x7FFFFFFFu) == 0u) u = 0u;
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

CC_DEV uint64_t slot_key(const float *s, int j, int n_sink) {
  const uint32_t k = j < n_sink ? kKeyPosInf : monotone_key(s[j]);
  return (uint64_t(k) << 32) | uint32_t(j);
}

// exclusive block scan of x (1024 threads); returns the exclusive prefix,
// *total = block sum.
CC_DEV int block_excl_scan(int x, int *wsum, int *total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int incl = x;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
    if (lane >= o) incl += y;
  }
  if (lane == 31) wsum[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    int w = wsum[lane], wi = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      int y = __shfl_up_sync(0xFFFFFFFFu, wi, o);
      if (lane >= o) wi += y;
    }
    wsum[lane] = wi - w;            // exclusive warp offsets
    if (lane == 31) wsum[32] = wi;  // block total
  }
  __syncthreads();
  const int r = incl - x + wsum[warp];
  *total = wsum[32];
  __syncthreads();
  return r;
}

__global__ void __launch_bounds__(kThreads, 1)
    select_kernel(const float *scores, const int32_t *seq_len, int cap, const int32_t *budget,
                  int n_sink, int32_t *keep_idx, int32_t *keep_count, unsigned *status) {
  __shared__ unsigned hist[256];
  __shared__ int wsum[33];
  __shared__ int s_digit, s_above, s_count;
  const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int n = seq_len[b];
  if (n < 0 || n > cap) {
    if (tid == 0) {
      set_status(status, CC_ERR_DEVICE_ARG);
      keep_count[b] = 0;
    }
    return;
  }
  const float *s = scores + (size_t)b * cap;
  int32_t *out = keep_idx + (size_t)b * cap;
  int J = budget[b];
  const int forced = min(n, 1 + max(n_sink, 0));
  if (J < forced) {
    if (tid == 0) set_status(status, CC_ERR_BUDGET);
    J = forced;
  }
  if (J >= n) {  // everything fits: identity
    for (int j = tid; j < n; j += kThreads) out[j] = j;
    if (tid == 0) keep_count[b] = n;
    return;
  }

  // ---- radix select of T = J-th largest key
  uint64_t prefix = 0;
  int k = J;
#pragma unroll 1
  for (int pass = 0; pass < 8; ++pass) {
    const int shift = 56 - 8 * pass;
    const uint64_t hi_mask = pass == 0 ? 0ull : (~0ull << (shift + 8));
    if (tid < 256) hist[tid] = 0;
    __syncthreads();
    for (int j = tid; j < n; j += kThreads) {
      const uint64_t key = slot_key(s, j, n_sink);
      if ((key & hi_mask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1u);
    }
    __syncthreads();
    if (warp == 0) {
      // lane l owns digits 255-8l down to 248-8l (descending)
      const int base = 255 - lane * 8;
      unsigned c[8], sum = 0;
#pragma unroll
      for (int e = 0; e < 8; ++e) { c[e] = hist[base - e]; sum += c[e]; }
      unsigned incl = sum;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        unsigned y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (lane >= o) incl += y;
      }
      const unsigned excl = incl - sum;
      if (excl < (unsigned)k && (unsigned)k <= incl) {
        unsigned run = excl;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          if (run + c[e] >= (unsigned)k) {
            s_digit = base - e;
            s_above = (int)run;
            s_count = (int)c[e];
            break;
          }
          run += c[e];
        }
      }
    }
    __syncthreads();
    prefix |= uint64_t(s_digit) << shift;
    k -= s_above;
    const bool settled = s_count == k;   // the whole bucket is kept
    __syncthreads();
    if (settled) break;
  }
  const uint64_t T = prefix;

  // ---- flag key >= T and emit the kept slots in ascending order
  int carry = 0;
  for (int base = 0; base < n; base += kThreads * 4) {
    const int j0 = base + tid * 4;
    int f[4], cnt = 0;
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int j = j0 + e;
      f[e] = (j < n && slot_key(s, j, n_sink) >= T) ? 1 : 0;
      cnt += f[e];
    }
    int total;
    int off = carry + block_excl_scan(cnt, wsum, &total);
#pragma unroll
    for (int e = 0; e < 4; ++e)
      if (f[e]) out[off++] = j0 + e;
    carry += total;
  }
  if (tid == 0) {
    keep_count[b] = J;
    if (carry != J) set_status(status, CC_ERR_DEVICE_ARG);   // cannot happen: keys are unique
  }
}

}  // namespace

cudaError_t launch_select(const float *scores, const int32_t *seq_len, int batch, int cap,
                          const int32_t *budget, int n_sink, int32_t *keep_idx,
                          int32_t *keep_count, unsigned *status, cudaStream_t st) {
  if (batch <= 0) return cudaSuccess;
  select_kernel<<<batch, kThreads, 0, st>>>(scores, seq_len, cap, budget, n_sink, keep_idx,
                                            keep_count, status);
  return cudaGetLastError();
}

}  // namespace cc
