// select.cuh -- keep-set selection kernel.
#pragma once
#include "cc_common.cuh"

namespace cc {

cudaError_t launch_select(const float *scores, const int32_t *seq_len, int batch, int cap,
                          const int32_t *budget, int n_sink, int32_t *keep_idx,
                          int32_t *keep_count, unsigned *status, cudaStream_t st);

}  // namespace cc
