// Host-side launch wrappers of the libkint kernels (internal to the library).
#pragma once
#include <cuda_runtime.h>
#include "kint_params.h"

namespace kint {

// Transposed (and, with split, tf32 hi/lo) copies of X [BH][T][d], one job per tensor:
//   nat_hi / nat_lo : [BH][T][d]   (only with split; may be null)
//   tr_hi  / tr_lo  : [BH][d][Tp]  (tr_lo only with split; tr_hi may be null)
//   dot             : [BH][T] row dot products X_t . Y_t (only when Y is non-null; Y then [BH][T][d])
struct PrepJob {
  const float* X;
  const float* Y;
  float *nat_hi, *nat_lo, *tr_hi, *tr_lo, *dot;
};
struct PrepJobs {
  PrepJob j[4];
  int n;
};
cudaError_t launch_prep(const PrepJobs& jobs, int BH, int T, int Tp, int d, bool split, cudaStream_t s);

cudaError_t launch_fwd_stats(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s);
cudaError_t launch_fwd_main(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s);
cudaError_t launch_bwd_dq(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s);
cudaError_t launch_bwd_dkdv(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s);

}  // namespace kint
