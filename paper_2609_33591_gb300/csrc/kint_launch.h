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
// Single-pass backward set-up, done by the job with Y (the dO job) for the rows it holds:
// the 16-byte row records {c0, 1/W, 1/W*, -<g>/W*} (position offset, forward
// normalizer, gamma = g / W* - <g> / W*; the softmax comparator keeps gamma = g - <g>),
// zeroed row sums and dQ rows, zeroed c_M / c_m outputs, and the 64-row query tiles of
// rows with tied maxima (tileflags) with the count of their tied keys (tie_total; tie_any
// set when that count exceeds tie_cap).  Inactive when frec is null.
struct RecJob {
  float4* frec;
  float *rsum, *dQ, *cM_out, *cm_out;
  const float *row_max, *W, *Ws;  // Ws: the W* of gamma (W_lerp under Prob-STE, else W)
  const int* n_max;
  int *tileflags, *tie_total, *tie_any;
  int nqt, tie_cap;
  int c0_kind;  // 0: c0 = -M log2(e); 1: FWM grids, (tau - M) / h (times 2 for the half-bin table: half); 2: -M
  int half, softmax;
  float tau, inv_h;
};
struct PrepJobs {
  PrepJob j[4];
  int n;
  RecJob rec;
};
// nsm: SMs of the device (the grid is a few CTAs per SM looping over the work units)
cudaError_t launch_prep(const PrepJobs& jobs, int BH, int T, int Tp, int d, bool split, int nsm, cudaStream_t s);

// Launch with programmatic stream serialization: the kernel may be scheduled while the
// previous kernel in the stream finishes; every kernel of the library waits for its
// predecessor (pdl_wait) before its first global access.
template <class Kern, class... Args>
cudaError_t launch_pdl(Kern kern, dim3 grid, dim3 block, int smem, cudaStream_t s, const Args&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = (size_t)smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}

// sch: the host item schedule of the persistent kernels (Sched::n == 0: snake order)
cudaError_t launch_fwd_stats(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s, const Sched& sch);
cudaError_t launch_fwd_main(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s, const Sched& sch);
cudaError_t launch_bwd_dq(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s);
cudaError_t launch_bwd_dkdv(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s);
// Geometry probe: per-row span, width, softmax entropy, share below -6, top-bucket mass,
// effective buckets and total variation to softmax, into p.probe
cudaError_t launch_fwd_probe(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s);
// Single-pass backward (TF32, d = 64; its row records come from the dO prep job, RecJob):
// the pass itself, and the extremum terms it leaves for afterwards
cudaError_t launch_bwd_fused(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s, const Sched& sch);
cudaError_t launch_bwd_ext(const Params& p, cudaStream_t s);
// C = running sums of the key rows of every head, [BH][T][d] (the P1 projection)
cudaError_t launch_kcum(const float* K, float* C, int BH, int T, int d, cudaStream_t s);

}  // namespace kint
