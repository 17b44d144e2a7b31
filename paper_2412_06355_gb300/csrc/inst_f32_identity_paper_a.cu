// Explicit instantiations of the fused DendSN kernels (forward and the backward with 4-step chunks): x dtype float32,
// psi = identity, the paper's (C_o, P, H, W) layer layout.
// One translation unit per (dtype, psi, layout, part) so the library builds in parallel.
#include "dendsn_kernels.cuh"

namespace dendsn {
#define DENDSN_INST(K, G) \
    template cudaError_t launch_forward<K, G, 0, 0, 1>(const FwdArgs &, int, cudaStream_t, int *);     \
    template cudaError_t launch_backward<K, G, 0, 0, 4, 1>(const BwdArgs &, int, cudaStream_t, int *);
DENDSN_KG_LIST(DENDSN_INST)
#undef DENDSN_INST
}  // namespace dendsn
