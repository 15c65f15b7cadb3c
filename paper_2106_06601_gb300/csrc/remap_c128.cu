// Remap kernels for double2 elements (see remap_impl.cuh).
#include "remap_impl.cuh"

namespace costa {

cudaError_t launch_remap_c128(const RemapLaunch &a, int kind, cudaStream_t st) {
    return remap::launch_remap_t<double2>(a, kind, st);
}

}  // namespace costa
