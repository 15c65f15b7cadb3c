// costa_volume_noalloc: the communication-volume count of costa_volume, for
// callers that must not have this library allocate device memory.
//
// Some callers cannot let a library call cudaMalloc: an application whose
// framework owns all device memory through its own pool (a cudaMalloc behind
// its back can fail under the pool's reservation or fragment it), and code
// on a latency-critical path, where cudaMalloc / cudaFree would synchronize
// the device.  This entry point therefore works only in a fixed scratch
// array that is part of the library's device image: a file-scope
// `static __device__` array of kScratchBytes (4 MiB), which every GPU that
// loads the library holds until the process exits.
//
// Host code must not use the array's name as a device address (on the host
// it names a stand-in); the address comes from cudaGetSymbolAddress, looked
// up by every call with the calling device current.  The lookup allocates
// nothing, and a fresh lookup stays right when the device's context has
// been created again (after cudaDeviceReset), which a cached address would
// not.
//
// Unlike costa_volume it builds no plan: one thread block per block of A
// finds, by binary search, the blocks of op(B) that overlap it, and its
// threads add the areas of those overlay cells to V (Alg. 2's package sizes).
// The result is the same exact integer matrix.
#include <cuda_runtime.h>

#include <cstdio>
#include <mutex>

#include "costa_internal.h"

namespace costa {
namespace {

constexpr size_t kScratchBytes = size_t(4) << 20;  // 4 MiB

static __device__ __align__(256) unsigned char g_noalloc_scratch[kScratchBytes];

std::mutex g_noalloc_mu;

// Last index k in [0, nb) with split[k] <= x (the block holding x; blocks
// that are empty share their start with the next one and are skipped).
__device__ __forceinline__ int last_le(const int64_t *split, int nb, int64_t x) {
    int lo = 0, hi = nb;
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (split[mid] <= x) lo = mid; else hi = mid;
    }
    return lo;
}

// One thread block per block (i, j) of A.  RBr / RBc are the row / column
// splits of op(B); owner of op(B) block (k, l) is ownB[k * nbcB + l] (N) or
// ownB[l * nbcB + k] (T, C).
__global__ void volume_noalloc_kernel(const int64_t *RA, const int64_t *CA, int nbrA, int nbcA,
                                      const int64_t *RBr, int nbr_op, const int64_t *RBc,
                                      int nbc_op, const int32_t *ownA, const int32_t *ownB,
                                      int nbcB, int transposed, int P, unsigned long long *V) {
    const int64_t b = blockIdx.x;
    const int i = static_cast<int>(b / nbcA), j = static_cast<int>(b - static_cast<int64_t>(i) * nbcA);
    const int64_t r0 = RA[i], r1 = RA[i + 1], c0 = CA[j], c1 = CA[j + 1];
    if (r1 <= r0 || c1 <= c0) return;
    const int q = ownA[b];
    const int k_lo = last_le(RBr, nbr_op, r0), k_hi = last_le(RBr, nbr_op, r1 - 1);
    const int l_lo = last_le(RBc, nbc_op, c0), l_hi = last_le(RBc, nbc_op, c1 - 1);
    const int nl = l_hi - l_lo + 1;
    const int64_t cells = static_cast<int64_t>(k_hi - k_lo + 1) * nl;
    for (int64_t t = threadIdx.x; t < cells; t += blockDim.x) {
        const int k = k_lo + static_cast<int>(t / nl), l = l_lo + static_cast<int>(t % nl);
        const int64_t rows = min(r1, RBr[k + 1]) - max(r0, RBr[k]);
        const int64_t cols = min(c1, RBc[l + 1]) - max(c0, RBc[l]);
        if (rows <= 0 || cols <= 0) continue;
        const int p = transposed ? ownB[static_cast<int64_t>(l) * nbcB + k]
                                 : ownB[static_cast<int64_t>(k) * nbcB + l];
        atomicAdd(V + static_cast<int64_t>(p) * P + q, static_cast<unsigned long long>(rows * cols));
    }
}

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

costa_status cuda_error(cudaError_t e, const char *what) {
    char msg[256];
    snprintf(msg, sizeof msg, "costa_volume_noalloc: %s: %s", what, cudaGetErrorString(e));
    return report_error(COSTA_ERR_CUDA, msg);
}

// An error after work was queued on `st`: wait for that work first, so that
// the next call (which may use another stream) cannot overlap it in the
// shared array; the wait's own status is not reported over the first error.
costa_status cuda_error_queued(cudaError_t e, const char *what, cudaStream_t st) {
    (void)cudaStreamSynchronize(st);
    return cuda_error(e, what);
}

}  // namespace
}  // namespace costa

using namespace costa;

extern "C" costa_status costa_volume_noalloc(costa_layout A, costa_layout B, costa_op op, int64_t *V,
                                             void *stream_v) {
    costa_status s = check_pair(A, B, op);
    if (s != COSTA_OK) return s;
    if (!V) return report_error(COSTA_ERR_INVALID_ARG, "costa_volume_noalloc: V is null");
    const int P = A->nranks;
    const bool tr = op != COSTA_OP_N;
    const std::vector<int64_t> &RBr = tr ? B->C : B->R;
    const std::vector<int64_t> &RBc = tr ? B->R : B->C;
    const int64_t nblkA = static_cast<int64_t>(A->nbr) * A->nbc;
    const int64_t nblkB = static_cast<int64_t>(B->nbr) * B->nbc;

    // scratch layout: V | RA | CA | RBr | RBc | ownerA | ownerB
    const size_t oV = 0;
    const size_t oRA = align256(oV + sizeof(unsigned long long) * P * P);
    const size_t oCA = align256(oRA + sizeof(int64_t) * A->R.size());
    const size_t oRBr = align256(oCA + sizeof(int64_t) * A->C.size());
    const size_t oRBc = align256(oRBr + sizeof(int64_t) * RBr.size());
    const size_t oOA = align256(oRBc + sizeof(int64_t) * RBc.size());
    const size_t oOB = align256(oOA + sizeof(int32_t) * nblkA);
    const size_t need = oOB + sizeof(int32_t) * nblkB;
    if (need > kScratchBytes || nblkA > 0x7fffffff) {
        char msg[256];
        snprintf(msg, sizeof msg,
                 "costa_volume_noalloc: this pair needs %zu bytes of scratch (P = %d, %lld + %lld "
                 "blocks); the fixed maximum is %zu bytes",
                 need, P, (long long)nblkA, (long long)nblkB, kScratchBytes);
        return report_error(COSTA_ERR_INVALID_ARG, msg);
    }

    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    // the array's address on the current device (in its current context)
    void *addr = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&addr, g_noalloc_scratch);
    if (e != cudaSuccess) return cuda_error(e, "cudaGetSymbolAddress");
    char *base = static_cast<char *>(addr);
    cudaStream_t st = static_cast<cudaStream_t>(stream_v);
    unsigned long long *dV = reinterpret_cast<unsigned long long *>(base + oV);

    // every call reuses the array: V must start from zero
    e = cudaMemsetAsync(dV, 0, sizeof(unsigned long long) * P * P, st);
    if (e != cudaSuccess) return cuda_error(e, "cudaMemsetAsync");
    struct Up { size_t off; const void *src; size_t bytes; } ups[] = {
        {oRA, A->R.data(), sizeof(int64_t) * A->R.size()},
        {oCA, A->C.data(), sizeof(int64_t) * A->C.size()},
        {oRBr, RBr.data(), sizeof(int64_t) * RBr.size()},
        {oRBc, RBc.data(), sizeof(int64_t) * RBc.size()},
        {oOA, A->owner.data(), sizeof(int32_t) * nblkA},
        {oOB, B->owner.data(), sizeof(int32_t) * nblkB},
    };
    for (const Up &u : ups) {
        if (!u.bytes) continue;
        e = cudaMemcpyAsync(base + u.off, u.src, u.bytes, cudaMemcpyHostToDevice, st);
        if (e != cudaSuccess) return cuda_error_queued(e, "cudaMemcpyAsync", st);
    }
    if (nblkA > 0) {
        volume_noalloc_kernel<<<static_cast<unsigned>(nblkA), 128, 0, st>>>(
            reinterpret_cast<const int64_t *>(base + oRA), reinterpret_cast<const int64_t *>(base + oCA),
            A->nbr, A->nbc, reinterpret_cast<const int64_t *>(base + oRBr),
            static_cast<int>(RBr.size()) - 1, reinterpret_cast<const int64_t *>(base + oRBc),
            static_cast<int>(RBc.size()) - 1, reinterpret_cast<const int32_t *>(base + oOA),
            reinterpret_cast<const int32_t *>(base + oOB), B->nbc, tr ? 1 : 0, P, dV);
        count_launch();
        e = cudaGetLastError();
        if (e != cudaSuccess) return cuda_error_queued(e, "kernel launch", st);
    }
    e = cudaMemcpyAsync(V, dV, sizeof(int64_t) * P * P, cudaMemcpyDeviceToHost, st);
    if (e != cudaSuccess) return cuda_error_queued(e, "cudaMemcpyAsync(V)", st);
    e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return cuda_error(e, "volume kernel");
    return COSTA_OK;
}
