// dK/dV kernels that also accumulate the per-row sums of dS and |dS| (a diagnostic
// side output of kint_attn_bwd: the zero-sum identity of Eq. (full) measured on the
// score gradient the dK contraction uses).  Their own translation unit, compiled in
// parallel with the plain ones.
#include "kint_bwd_kv.cuh"

namespace kint {

template cudaError_t launch_bwd_dkdv_t<true>(const Maps&, const Params&, int, cudaStream_t);

}  // namespace kint
