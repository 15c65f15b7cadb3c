// Grid-overlay volume kernel (Alg. 2) and the remap launch dispatcher.
//
// The overlay of L(A) and L(op(B)) is the product of row intervals and
// column intervals (Sec. 5, "Grid Overlay"); one thread per overlay cell adds
// the cell's area to V[owner in L(B)][owner in L(A)] with a 64-bit atomic.
// Integer sums are exact and order-independent, so V is deterministic.
#include <cuda_runtime.h>

#include <atomic>
#include <cstdint>

#include "costa_internal.h"

namespace costa {

namespace {

std::atomic<int64_t> g_launches{0};

// ---- grid-overlay volume (Alg. 2): one thread per overlay cell ----
__global__ void volume_kernel(const VolumeLaunch a) {
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t t = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; t < a.total_cells;
         t += stride) {
        int k = 0;
        if (a.nprob > 1) {
            int lo = 0, hi = a.nprob;
            while (hi - lo > 1) {
                const int mid = (lo + hi) >> 1;
                if (a.probs[mid].cell_begin <= t) lo = mid; else hi = mid;
            }
            k = lo;
        }
        const VolumeProblemDev &P = a.probs[k];
        const int64_t tl = t - P.cell_begin;
        const int r = static_cast<int>(tl / P.nc);
        const int c = static_cast<int>(tl - static_cast<int64_t>(r) * P.nc);
        const Interval ri = P.rows[r];
        const Interval ci = P.cols[c];
        const int q = P.ownerA[static_cast<int64_t>(ri.a_blk) * P.nbcA + ci.a_blk];
        const int p = P.op == COSTA_OP_N ? P.ownerB[static_cast<int64_t>(ri.b_blk) * P.nbcB + ci.b_blk]
                                         : P.ownerB[static_cast<int64_t>(ci.b_blk) * P.nbcB + ri.b_blk];
        atomicAdd(a.V + static_cast<int64_t>(p) * a.P + q,
                  static_cast<unsigned long long>(ri.len * ci.len));
    }
}

int sm_count() {
    static int cached = 0;
    if (!cached) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&cached, cudaDevAttrMultiProcessorCount, dev);
        if (cached <= 0) cached = 1;
    }
    return cached;
}

}  // namespace

void count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

int64_t launches_so_far() { return g_launches.load(std::memory_order_relaxed); }

cudaError_t launch_remap(const RemapLaunch &a, int kind, cudaStream_t stream) {
    if (a.ntiles <= 0 && a.nmtiles <= 0 && a.ngroups <= 0 && !(a.tma && a.tma->nttiles > 0)) return cudaSuccess;
    switch (a.dtype) {
    case COSTA_F32: return launch_remap_f32(a, kind, stream);
    case COSTA_F64: return launch_remap_f64(a, kind, stream);
    case COSTA_C64: return launch_remap_c64(a, kind, stream);
    case COSTA_C128: return launch_remap_c128(a, kind, stream);
    default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_volume(const VolumeLaunch &a, cudaStream_t stream) {
    if (a.total_cells <= 0) return cudaSuccess;
    const int threads = 256;
    const int64_t want = (a.total_cells + threads - 1) / threads;
    const int64_t cap = static_cast<int64_t>(sm_count()) * 8;
    const int blocks = static_cast<int>(want < cap ? want : cap);
    volume_kernel<<<blocks, threads, 0, stream>>>(a);
    count_launch();
    return cudaGetLastError();
}

}  // namespace costa
