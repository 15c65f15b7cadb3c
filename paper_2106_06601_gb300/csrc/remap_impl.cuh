// Remap kernels of the reshuffle A = alpha * op(B) + beta * A (Eq. 1, Sec. 5),
// templated on the element type; each element type is compiled in its own
// translation unit (remap_f32.cu, remap_f64.cu, remap_c64.cu, remap_c128.cu).
//
// Work decomposition.  The grid overlay of L(A) and L(op(B)) (Sec. 5, "Grid
// Overlay") is the product of row intervals and column intervals; the host
// cuts each interval into pieces of at most TS elements, so the kernel's tile
// grid is (row pieces) x (column pieces), and every tile lies inside one block
// of A and one block of B.  Inside a tile both storages are affine, so one
// warp moves it with 16-byte vector accesses where alignment allows:
//   - if A and the source share their contiguous axis, the warp copies runs
//     straight through registers;
//   - otherwise it transposes through a padded shared-memory tile (Sec. 6:
//     "cache-friendly ... kernel for matrix transposition"): source runs in,
//     target runs out, with alpha / beta applied as one fma on the way out
//     (Sec. 5: transform after receive).
// Warps sweep the tile list in a grid-stride loop over a persistent grid.
//
// Modes: DIRECT_ALL (B -> A for every tile), and the message path of Alg. 3 /
// Sec. 6: PACK (remote tiles: B -> staging, an exact copy), DIRECT_LOCAL
// (tiles local after relabeling: B -> A), UNPACK (remote tiles: staging -> A
// with the transform).
//
// No kernel here waits on another block or on a flag: there are no
// spin-waits, so no wait can fail to end.

#pragma once

#include <cuda_runtime.h>

#include <cstdint>

#include "costa_internal.h"

namespace costa {
namespace remap {

template <typename T> struct ET;
template <> struct ET<float>   { enum { VEC = 4, CPLX = 0 }; typedef float R; };
template <> struct ET<double>  { enum { VEC = 2, CPLX = 0 }; typedef double R; };
template <> struct ET<float2>  { enum { VEC = 2, CPLX = 1 }; typedef float R; };
template <> struct ET<double2> { enum { VEC = 1, CPLX = 1 }; typedef double R; };

// Per element type: tile extent TS, 16-byte chunk width VEC (elements), and
// the lane mapping: CPR chunks cover one run of TS elements, a warp pass
// covers RPP runs, NPASS passes cover TS runs.
template <typename T> struct Cfg {
    static constexpr int TS = sizeof(T) == 16 ? 16 : 32;
    static constexpr int VEC = ET<T>::VEC;
    static constexpr int CPR = TS / VEC;
    static constexpr int RPP = 32 / CPR;
    static constexpr int NPASS = TS / RPP;
    static constexpr int PITCH = TS + 1;  // odd pitch: conflict-light columns
    static constexpr int SMEM_ELEMS = TS * PITCH;
};
constexpr int kWarps = 8;

template <typename T> struct Chunk {
    union {
        uint4 raw;
        T e[ET<T>::VEC];
    };
};

template <typename T>
__device__ __forceinline__ Chunk<T> load_ro(const T *p) {
    Chunk<T> c;
    c.raw = __ldg(reinterpret_cast<const uint4 *>(p));
    return c;
}

template <typename T>
__device__ __forceinline__ Chunk<T> load_rw(const T *p) {
    Chunk<T> c;
    c.raw = *reinterpret_cast<const uint4 *>(p);
    return c;
}

template <typename T>
__device__ __forceinline__ void store(T *p, const Chunk<T> &c) {
    *reinterpret_cast<uint4 *>(p) = c.raw;
}

// ---- alpha * b + beta * a, one rounding per fma (no contraction freedom) ----
__device__ __forceinline__ float mulr(float a, float b) { return __fmul_rn(a, b); }
__device__ __forceinline__ double mulr(double a, double b) { return __dmul_rn(a, b); }
__device__ __forceinline__ float fmar(float a, float b, float c) { return __fmaf_rn(a, b, c); }
__device__ __forceinline__ double fmar(double a, double b, double c) { return __fma_rn(a, b, c); }

struct Sc {
    double ar, ai, br, bi;
    uint32_t conj_mask;  // 0x80000000 flips the sign of b's imaginary part (op = C)
};

// Combine of one element for a kind K_* (costa_internal.h); the kernel is
// compiled per kind.  b arrives conjugated (op = C) via conj_mask.

template <int KIND, typename R>
__device__ __forceinline__ R comb_real(R b, R a, const Sc &s) {
    if (KIND == K_COPY) return b;
    if (KIND == K_SCALE) return mulr(R(s.ar), b);
    return fmar(R(s.ar), b, mulr(R(s.br), a));
}

template <int KIND>
__device__ __forceinline__ float combine(float b, float a, const Sc &s) { return comb_real<KIND, float>(b, a, s); }
template <int KIND>
__device__ __forceinline__ double combine(double b, double a, const Sc &s) { return comb_real<KIND, double>(b, a, s); }

__device__ __forceinline__ float flip_sign(float v, uint32_t m) {
    return __uint_as_float(__float_as_uint(v) ^ m);
}
__device__ __forceinline__ double flip_sign(double v, uint32_t m) {
    return __longlong_as_double(__double_as_longlong(v) ^ (static_cast<unsigned long long>(m) << 32));
}

template <int KIND, typename C, typename R>
__device__ __forceinline__ C combine_c(C b, C a, const Sc &s) {
    b.y = flip_sign(b.y, s.conj_mask);
    C o;
    if (KIND != K_CPLX) {
        o.x = comb_real<KIND, R>(b.x, a.x, s);
        o.y = comb_real<KIND, R>(b.y, a.y, s);
        return o;
    }
    const R ar = R(s.ar), ai = R(s.ai), br = R(s.br), bi = R(s.bi);
    R t = fmar(br, a.x, -mulr(bi, a.y));
    t = fmar(-ai, b.y, t);
    o.x = fmar(ar, b.x, t);
    R w = fmar(br, a.y, mulr(bi, a.x));
    w = fmar(ai, b.x, w);
    o.y = fmar(ar, b.y, w);
    return o;
}
template <int KIND>
__device__ __forceinline__ float2 combine(float2 b, float2 a, const Sc &s) {
    return combine_c<KIND, float2, float>(b, a, s);
}
template <int KIND>
__device__ __forceinline__ double2 combine(double2 b, double2 a, const Sc &s) {
    return combine_c<KIND, double2, double>(b, a, s);
}

// A tile in its canonical frame: x = the target's contiguous axis.
//   target element (x, y) at dst + x + y * dld
//   source element (x, y) at src + x + y * sld        (copy tile)
//                         or src + x * sld + y        (transposed tile)
template <typename T> struct Geom {
    T *dst;
    const T *src;
    int64_t dld, sld;
    int nx, ny;
    bool transpose, dvec, svec;
};

// Fast paths: every chunk is a full, 16-byte aligned vector (checked by the
// caller), so the unrolled loops carry no element-level branches.

template <typename T, int KIND>
__device__ __forceinline__ void tile_copy_vec(const Geom<T> &g, const Sc &s, int lane) {
    constexpr bool READ_A = KIND >= K_AXPBY;
    using C = Cfg<T>;
    constexpr int G = C::NPASS > 8 ? 8 : C::NPASS;  // passes in flight per group
    const int c = lane % C::CPR, yr = lane / C::CPR, x0 = c * C::VEC;
    const bool lane_on = x0 < g.nx;
#pragma unroll
    for (int p0 = 0; p0 < C::NPASS; p0 += G) {
        Chunk<T> bv[G], av[G];
#pragma unroll
        for (int p = 0; p < G; ++p) {
            av[p].raw = make_uint4(0, 0, 0, 0);
            const int y = (p0 + p) * C::RPP + yr;
            if (lane_on && y < g.ny) {
                bv[p] = load_ro(g.src + y * g.sld + x0);
                if (READ_A) av[p] = load_rw(g.dst + y * g.dld + x0);
            }
        }
#pragma unroll
        for (int p = 0; p < G; ++p) {
            const int y = (p0 + p) * C::RPP + yr;
            if (lane_on && y < g.ny) {
                Chunk<T> o;
#pragma unroll
                for (int e = 0; e < C::VEC; ++e) o.e[e] = combine<KIND>(bv[p].e[e], av[p].e[e], s);
                store(g.dst + y * g.dld + x0, o);
            }
        }
    }
}

template <typename T, int KIND>
__device__ __forceinline__ void tile_transpose_vec(const Geom<T> &g, const Sc &s, T *sm, int lane) {
    using C = Cfg<T>;
    constexpr bool READ_A = KIND >= K_AXPBY;
    constexpr int G = C::NPASS > 8 ? 8 : C::NPASS;  // target passes per group
    {   // source runs (along y) -> sm[y][x]
        const int c = lane % C::CPR, xr = lane / C::CPR, y0 = c * C::VEC;
        const bool lane_on = y0 < g.ny;
#pragma unroll
        for (int p0 = 0; p0 < C::NPASS; p0 += G) {
            Chunk<T> bv[G];
#pragma unroll
            for (int p = 0; p < G; ++p) {
                const int x = (p0 + p) * C::RPP + xr;
                if (lane_on && x < g.nx) bv[p] = load_ro(g.src + x * g.sld + y0);
            }
#pragma unroll
            for (int p = 0; p < G; ++p) {
                const int x = (p0 + p) * C::RPP + xr;
                if (lane_on && x < g.nx) {
#pragma unroll
                    for (int e = 0; e < C::VEC; ++e) sm[(y0 + e) * C::PITCH + x] = bv[p].e[e];
                }
            }
        }
    }
    __syncwarp();
    {   // target runs (along x) <- sm[y][x], combined with A
        const int c = lane % C::CPR, yr = lane / C::CPR, x0 = c * C::VEC;
        const bool lane_on = x0 < g.nx;
#pragma unroll
        for (int p0 = 0; p0 < C::NPASS; p0 += G) {
            Chunk<T> av[G];
#pragma unroll
            for (int p = 0; p < G; ++p) {
                av[p].raw = make_uint4(0, 0, 0, 0);
                const int y = (p0 + p) * C::RPP + yr;
                if (READ_A && lane_on && y < g.ny) av[p] = load_rw(g.dst + y * g.dld + x0);
            }
#pragma unroll
            for (int p = 0; p < G; ++p) {
                const int y = (p0 + p) * C::RPP + yr;
                if (lane_on && y < g.ny) {
                    Chunk<T> o;
#pragma unroll
                    for (int e = 0; e < C::VEC; ++e)
                        o.e[e] = combine<KIND>(sm[y * C::PITCH + x0 + e], av[p].e[e], s);
                    store(g.dst + y * g.dld + x0, o);
                }
            }
        }
    }
    __syncwarp();
}

// General path for ragged or misaligned tiles: element by element, lanes
// strided along the contiguous axis of each phase.
template <typename T, int KIND>
__device__ __forceinline__ void tile_general(const Geom<T> &g, const Sc &s, T *sm, int lane) {
    using C = Cfg<T>;
    constexpr bool READ_A = KIND >= K_AXPBY;
    const int n = g.nx * g.ny;
    if (!g.transpose) {
        for (int k = lane; k < n; k += 32) {
            const int y = k / g.nx, x = k - y * g.nx;
            T *d = g.dst + y * g.dld + x;
            const T a = READ_A ? *d : T();
            *d = combine<KIND>(__ldg(g.src + y * g.sld + x), a, s);
        }
        return;
    }
    for (int k = lane; k < n; k += 32) {
        const int x = k / g.ny, y = k - x * g.ny;
        sm[y * C::PITCH + x] = __ldg(g.src + x * g.sld + y);
    }
    __syncwarp();
    for (int k = lane; k < n; k += 32) {
        const int y = k / g.nx, x = k - y * g.nx;
        T *d = g.dst + y * g.dld + x;
        const T a = READ_A ? *d : T();
        *d = combine<KIND>(sm[y * C::PITCH + x], a, s);
    }
    __syncwarp();
}

template <typename T, int KIND>
__device__ __forceinline__ void run_tile(const Geom<T> &g, const Sc &s, T *sm, int lane) {
    using C = Cfg<T>;
    // vector fast path: both sides 16-byte aligned and every run a whole
    // number of chunks (the source runs along y when transposing)
    const int vrun_src = g.transpose ? g.ny : g.nx;
    const bool fast = g.dvec && g.svec && (g.nx % C::VEC) == 0 && (vrun_src % C::VEC) == 0;
    if (!fast) tile_general<T, KIND>(g, s, sm, lane);
    else if (g.transpose) tile_transpose_vec<T, KIND>(g, s, sm, lane);
    else tile_copy_vec<T, KIND>(g, s, lane);
}

__device__ __forceinline__ bool aligned16(const void *p, int64_t ld_bytes) {
    return ((reinterpret_cast<uintptr_t>(p) | static_cast<uintptr_t>(ld_bytes)) & 15) == 0;
}

template <typename T, int MODE, int KIND>
__global__ void __launch_bounds__(kWarps * 32, 2) remap_kernel(const RemapLaunch args) {
    using C = Cfg<T>;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    T *sm = reinterpret_cast<T *>(smem_raw) + warp * C::SMEM_ELEMS;
    const int64_t nwarps = static_cast<int64_t>(gridDim.x) * kWarps;

    for (int64_t t = static_cast<int64_t>(blockIdx.x) * kWarps + warp; t < args.total_tiles;
         t += nwarps) {
        int k = 0;
        if (args.nprob > 1) {
            int lo = 0, hi = args.nprob;
            while (hi - lo > 1) {
                const int mid = (lo + hi) >> 1;
                if (args.probs[mid].tile_begin <= t) lo = mid; else hi = mid;
            }
            k = lo;
        }
        const ProblemDev &P = args.probs[k];
        const int64_t tl = t - P.tile_begin;
        int64_t soff = -1;
        int64_t stld = 0;
        if (MODE != KM_DIRECT_ALL) {
            soff = P.stage_off[tl];
            if (MODE == KM_DIRECT_LOCAL ? soff >= 0 : soff < 0) continue;
            stld = P.stage_ld[tl];
        }
        const int u = static_cast<int>(tl / P.nv);
        const int v = static_cast<int>(tl - static_cast<int64_t>(u) * P.nv);
        const AxisTile rt = P.rows[u];
        const AxisTile ct = P.cols[v];
        const DevBlock dA = P.descA[static_cast<int64_t>(rt.a_blk) * P.nbcA + ct.a_blk];
        const int op = P.op;
        const DevBlock dB = op == COSTA_OP_N
                                ? P.descB[static_cast<int64_t>(rt.b_blk) * P.nbcB + ct.b_blk]
                                : P.descB[static_cast<int64_t>(ct.b_blk) * P.nbcB + rt.b_blk];

        // source block element (rb, cb) of tile element (i, j)
        const bool b_col = dB.order == COSTA_COL_MAJOR;
        int64_t rb, cb;
        bool src_fast_i;
        if (op == COSTA_OP_N) { rb = rt.b_off; cb = ct.b_off; src_fast_i = b_col; }
        else                  { rb = ct.b_off; cb = rt.b_off; src_fast_i = !b_col; }
        const T *src = reinterpret_cast<const T *>(dB.ptr) + (b_col ? rb + cb * dB.ld : rb * dB.ld + cb);
        int64_t sld = dB.ld;

        const bool a_col = dA.order == COSTA_COL_MAJOR;
        T *dst = reinterpret_cast<T *>(dA.ptr) +
                 (a_col ? rt.a_off + static_cast<int64_t>(ct.a_off) * dA.ld
                        : static_cast<int64_t>(rt.a_off) * dA.ld + ct.a_off);
        int64_t dld = dA.ld;
        bool dst_fast_i = a_col;

        if (MODE == KM_PACK) {
            dst = reinterpret_cast<T *>(args.staging) + soff;
            dld = stld;
            dst_fast_i = src_fast_i;
        } else if (MODE == KM_UNPACK) {
            src = reinterpret_cast<const T *>(args.staging) + soff;
            sld = stld;
        }

        Geom<T> g;
        g.dst = dst;
        g.src = src;
        g.dld = dld;
        g.sld = sld;
        g.nx = dst_fast_i ? rt.len : ct.len;
        g.ny = dst_fast_i ? ct.len : rt.len;
        g.transpose = dst_fast_i != src_fast_i;
        g.dvec = aligned16(dst, dld * static_cast<int64_t>(sizeof(T)));
        g.svec = aligned16(src, sld * static_cast<int64_t>(sizeof(T)));

        Sc s{1.0, 0.0, 0.0, 0.0, 0u};
        if (MODE != KM_PACK) {
            Scalars S;
            if (args.per_problem) {
                S = args.per_problem[k];
                if (kind_of(S.flags) != KIND) continue;  // another launch covers it
            } else {
                S = args.s;
            }
            s.ar = S.alpha[0]; s.ai = S.alpha[1]; s.br = S.beta[0]; s.bi = S.beta[1];
            s.conj_mask = (ET<T>::CPLX && op == COSTA_OP_C) ? 0x80000000u : 0u;
        }
        run_tile<T, KIND>(g, s, sm, lane);
    }
}

inline int sm_count() {
    static int cached = 0;
    if (!cached) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&cached, cudaDevAttrMultiProcessorCount, dev);
        if (cached <= 0) cached = 1;
    }
    return cached;
}

template <typename T, int MODE, int KIND>
cudaError_t launch_t(const RemapLaunch &a, cudaStream_t st) {
    auto kern = remap_kernel<T, MODE, KIND>;
    const size_t smem = static_cast<size_t>(kWarps) * Cfg<T>::SMEM_ELEMS * sizeof(T);
    static int per_sm = 0;
    if (per_sm == 0) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(smem));
        if (e != cudaSuccess) return e;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kWarps * 32, smem);
        if (e != cudaSuccess) return e;
        if (per_sm < 1) per_sm = 1;
    }
    const int64_t want = (a.total_tiles + kWarps - 1) / kWarps;
    const int64_t cap = static_cast<int64_t>(sm_count()) * per_sm;
    const int blocks = static_cast<int>(want < cap ? want : cap);
    if (blocks <= 0) return cudaSuccess;
    kern<<<blocks, kWarps * 32, smem, st>>>(a);
    count_launch();
    return cudaGetLastError();
}

// Kernel for (element type, mode, combine kind).  Real types never take
// K_CPLX; PACK is always a plain copy.
template <typename T>
cudaError_t launch_remap_t(const RemapLaunch &a, int mode, int kind, cudaStream_t st) {
    if (mode == KM_PACK) return launch_t<T, KM_PACK, K_COPY>(a, st);
#define COSTA_KINDS(MODE)                                                         \
    switch (kind) {                                                               \
    case K_COPY: return launch_t<T, MODE, K_COPY>(a, st);                         \
    case K_SCALE: return launch_t<T, MODE, K_SCALE>(a, st);                       \
    case K_AXPBY: return launch_t<T, MODE, K_AXPBY>(a, st);                       \
    default:                                                                      \
        if (ET<T>::CPLX) return launch_t<T, MODE, K_CPLX>(a, st);                 \
        return cudaErrorInvalidValue;                                             \
    }
    switch (mode) {
    case KM_DIRECT_ALL: COSTA_KINDS(KM_DIRECT_ALL)
    case KM_DIRECT_LOCAL: COSTA_KINDS(KM_DIRECT_LOCAL)
    case KM_UNPACK: COSTA_KINDS(KM_UNPACK)
    default: return cudaErrorInvalidValue;
    }
#undef COSTA_KINDS
}

}  // namespace remap
}  // namespace costa
