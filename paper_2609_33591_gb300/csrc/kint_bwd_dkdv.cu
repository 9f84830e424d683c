// dK/dV kernels of the backward (App. B): the plain instantiations, and the launch
// entry that picks them or the row-sum ones (kint_bwd_dkdv_rs.cu).
#include "kint_bwd_kv.cuh"

namespace kint {

extern template cudaError_t launch_bwd_dkdv_t<true>(const Maps&, const Params&, int, cudaStream_t);
template cudaError_t launch_bwd_dkdv_t<false>(const Maps&, const Params&, int, cudaStream_t);

cudaError_t launch_bwd_dkdv(const Maps& maps, const Params& p, int smem_bytes, cudaStream_t s) {
  if (p.dsum_out || p.dabs_out) return launch_bwd_dkdv_t<true>(maps, p, smem_bytes, s);
  return launch_bwd_dkdv_t<false>(maps, p, smem_bytes, s);
}

}  // namespace kint
