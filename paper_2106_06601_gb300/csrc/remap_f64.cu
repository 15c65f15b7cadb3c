// Remap kernels for double elements (see remap_impl.cuh).
#include "remap_impl.cuh"

namespace costa {

cudaError_t launch_remap_f64(const RemapLaunch &a, int kind, cudaStream_t st) {
    return remap::launch_remap_t<double>(a, kind, st);
}

}  // namespace costa
