// Remap kernels for float elements (see remap_impl.cuh).
#include "remap_impl.cuh"

namespace costa {

cudaError_t launch_remap_f32(const RemapLaunch &a, int kind, cudaStream_t st) {
    return remap::launch_remap_t<float>(a, kind, st);
}

}  // namespace costa
