// Host-side launch wrappers of the libkint kernels (internal to the library).
#pragma once
#include <cuda_runtime.h>
#include "kint_params.h"

namespace kint {

// Transposed (and, with split, tf32 hi/lo) copies of X [BH][T][d]:
//   nat_hi / nat_lo : [BH][T][d]   (only with split; may be null)
//   tr_hi  / tr_lo  : [BH][d][Tp]  (tr_lo only with split; tr_hi may be null)
//   dot             : [BH][T] row dot products X_t . Y_t (only when non-null; Y then [BH][T][d])
cudaError_t launch_prep(const float* X, float* nat_hi, float* nat_lo, float* tr_hi, float* tr_lo, int BH, int T,
                        int Tp, int d, bool split, cudaStream_t s, const float* Y = nullptr, float* dot = nullptr);

cudaError_t launch_fwd_stats(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s);
cudaError_t launch_fwd_main(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s);
cudaError_t launch_bwd_dq(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s);
cudaError_t launch_bwd_dkdv(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s);

}  // namespace kint
