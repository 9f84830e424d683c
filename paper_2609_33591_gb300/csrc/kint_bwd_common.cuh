// Shared pieces of the backward kernels (App. B): tile size, constants and the
// launch helper.  Included by the dQ and dK/dV translation units.
#pragma once
#include <cfloat>
#include "kint_dev.cuh"
#include "kint_launch.h"

namespace kint {

constexpr int BT = 64;  // keys per tile (k_bwd_dq), queries per tile (k_bwd_dkdv)

__device__ __forceinline__ int4 lds_i4(uint32_t addr) {
  int4 v;
  asm volatile("ld.shared.v4.s32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
  return v;
}

template <class K>
static cudaError_t launch3(K kern, dim3 grid, const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s,
                           int nthr = NTHR) {
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes);
  if (e != cudaSuccess) return e;
  return launch_pdl(kern, grid, dim3(nthr), smem_bytes, s, maps, p);
}

}  // namespace kint
