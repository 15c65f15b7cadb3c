// Remap kernels for float2 elements (see remap_impl.cuh).
#include "remap_impl.cuh"

namespace costa {

cudaError_t launch_remap_c64(const RemapLaunch &a, int kind, cudaStream_t st) {
    return remap::launch_remap_t<float2>(a, kind, st);
}

}  // namespace costa
