// Remap kernels of the reshuffle A = alpha * op(B) + beta * A (Eq. 1, Sec. 5),
// templated on the element type; each element type is compiled in its own
// translation unit (remap_f32.cu, remap_f64.cu, remap_c64.cu, remap_c128.cu).
//
// Work decomposition.  The grid overlay of L(A) and L(op(B)) (Sec. 5, "Grid
// Overlay") is the product of row intervals and column intervals; the host
// cuts each interval into pieces of at most TS elements, so the kernel's tile
// grid is (row pieces) x (column pieces), and every tile lies inside one block
// of A and one block of B.  Inside a tile both storages are affine.
//
// One warp moves one tile at a time, in a software pipeline over its tiles:
//   1. the source tile is staged into shared memory with 16-byte cp.async
//      copies (no registers held while in flight), one run of the source's
//      contiguous axis per shared-memory row, chunks XOR-swizzled per row so
//      that reading it transposed is free of avoidable bank conflicts;
//   2. while that is in flight the warp issues the copies of its next tile
//      into the other buffer and, when beta != 0, loads its A chunks into
//      registers;
//   3. it then writes A in A's contiguous order, 16 bytes per lane, applying
//      alpha and beta as one fma per element on the way out (Sec. 5:
//      transform after receive).
// If A and the source share their contiguous axis the staged rows are read
// straight; otherwise they are read across rows (the transposing kernel of
// Sec. 6).  Tiles whose runs are not 16-byte aligned take the same pipeline
// in a second instance of the kernel: over aligned 16-byte windows of their
// runs, or one element per lane (the kinds that read A, and 4-byte tiles
// whose target runs are misaligned).  A third instance stages the aligned
// source tiles of one kind (f64, general beta) by TMA, and a separate
// kernel moves lists of small tiles as grouped one-pass pieces.
//
// "alpha and beta as one fma" holds for real scalars; complex scalars take
// a compensated evaluation per component (Dot2; for double data Kahan's
// algorithm when a component has two terms, and a fixed-point sum on the
// integer pipes when it has four), see combine_c.
//
// The kernel walks a list of tile descriptors (TileDesc) resolved on the host:
// the direct list (every tile: B -> A), or the message path of Alg. 3 /
// Sec. 6 as three lists: pack (remote tiles: B -> staging, an exact copy,
// launched as K_COPY), local (tiles local after relabeling: B -> A) and
// unpack (remote tiles: staging -> A with the transform).  Each warp takes
// every (gridDim.x * warps)-th tile and reads the descriptors 32 at a time.
//
// No kernel here waits on another block or on a flag.  cp.async.wait_group
// waits only for this thread's own copies, which always complete.

#pragma once

#include <cuda_runtime.h>

#include <cstdint>

#include "costa_internal.h"
#include "fxdot.h"

namespace costa {
namespace remap {

template <typename T> struct ET;
template <> struct ET<float>   { enum { VEC = 4, CPLX = 0 }; typedef float R; };
template <> struct ET<double>  { enum { VEC = 2, CPLX = 0 }; typedef double R; };
template <> struct ET<float2>  { enum { VEC = 2, CPLX = 1 }; typedef float R; };
template <> struct ET<double2> { enum { VEC = 1, CPLX = 1 }; typedef double R; };

// Launch shape of the tile kernel per element size, combine kind and
// instance, all measured on GB300 (same box, 8192^2, GB/s): warps per
// block, the resident blocks per SM that the registers must allow (MINB),
// and shared-memory buffers per warp (NBUF: a warp keeps NBUF - 1 tiles'
// copies in flight ahead of the tile it writes).
//
//   element  instance     kinds                         warps  MINB  NBUF
//   4-byte   both         copy, scale                     8      2     2
//            both         kinds that read A               8      3     1
//   8-byte   aligned      copy, axpby2 (beta = +-2^k)     4      5     1
//            aligned      f64 scale                       4      2     3
//            aligned      c64 scale                       4      5     1
//            both         real general beta               4      3     2
//            both         complex beta                    4      4     1
//            both         complex alpha, beta = 0         4      2     3
//            misaligned   copy (16-byte windows)          4      5     3
//            misaligned   scale (16-byte windows)         4      5     2
//            misaligned   axpby2 (one element per lane)   4      4     1
//   16-byte  both         copy                            4      1     2
//            both         scale                           4      3     1
//            both         complex alpha, beta = 0         4      3     1
//            both         kinds that read A               4      2     1
//
// Why, where a row departs from its neighbours:
//  - 8-byte light kinds (copy, axpby2) run more warps without look-ahead;
//    the real general kind needs the registers of 3 blocks.
//  - f64 and c128 scale: one multiply per element on the narrow FP64 pipe,
//    hidden by more tiles in flight than the copy has: f64 T alpha=2 5400
//    -> 6204, N alpha=-0.7 5361 -> 6147 (the copy's rate) with two tiles
//    ahead; c128 T 4410 -> 5853, N 4343 -> 5746 with 3 blocks.  c64
//    (float multiplies) lost 11% with f64's shape and keeps the light one.
//    c128 with a complex alpha (FP64-bound at 8 operations per element
//    with Kahan's algorithm alone): T and N 1458 -> 2133 with 2 to 4
//    blocks; with every other element summed in fixed point on the integer
//    pipes (COSTA_FX_CS_PERIOD), unrolled, 2557 at 2 blocks, 2660 at 3 (one
//    pass in 3 or 4 in fixed point: 2553, 2569); in the rolled loop, 3 blocks,
//    3259.
//  - c64 complex scalars, against 3 blocks with 2 buffers: complex beta
//    T 4484 -> 5482, N 4495 -> 5495 with 4 blocks and no look-ahead;
//    complex alpha T 5551 -> 5955 with two tiles ahead; the real general
//    kind loses with either (6492 -> 6400 and 6082).
//  - 8-byte window path (misaligned instance, kinds that do not read A):
//    an 8.5 KB buffer per tile, so shared memory, not MINB, sets the blocks
//    per SM (6 with 1 buffer, 3 with 2, 2 with 3).  One tile ahead took f64
//    BC50 -> BC75 copy 3820 -> 4101, scale 3620 -> 4162, c64 copy 3797 ->
//    4093 (odd leading dimensions -0.4 to +1%); two tiles ahead took the
//    copy further (BC50 -> BC75 4518 -> 4677, BC75 -> BC75 4468 -> 5237,
//    BC64 -> BC75 5050 -> 5380, c64 BC50 -> BC75 4534 -> 4755; odd lds
//    -1.5 to +0.4%) but cost the scale kind 17%, whose FP64 multiplies 8
//    warps per SM leave exposed; 4 buffers lost 20-40%.
//  - 8-byte element path (misaligned, kinds that read A): a whole tile of A
//    in registers, which 4 blocks fit without spills.
//  - 16-byte kinds that read A hold a whole 16 KB tile of A in registers,
//    except with a complex beta: there each component is a fixed-point sum
//    on the integer pipes (498 GB/s with Dot2 on the FP64 pipe), and the
//    drain is a rolled loop over COSTA_FX_GROUP passes at a time that loads
//    A two groups ahead (unrolled with A's tile in registers: 1105 one pass
//    at a time, 1186 with 2, 1194 with 4, instruction fetch the limit;
//    rolled: 2286 with 1, 2340 with 2 at 136 registers and 3 blocks, 2115
//    with 4).
// Each entry is overridable at build time for tuning (COSTA_WARPS_4/8,
// COSTA_MINB_* and COSTA_NBUF_*).
#ifndef COSTA_WARPS_4
#define COSTA_WARPS_4 8
#endif
#ifndef COSTA_WARPS_8
#define COSTA_WARPS_8 4
#endif
// 4-byte: light kinds, kinds that read A
#ifndef COSTA_MINB_4
#define COSTA_MINB_4 2
#endif
#ifndef COSTA_NBUF_4
#define COSTA_NBUF_4 2
#endif
#ifndef COSTA_MINB_4A
#define COSTA_MINB_4A 3
#endif
#ifndef COSTA_NBUF_4A
#define COSTA_NBUF_4A 1
#endif
// 8-byte: light kinds (L), f64 scale (S), real general (H), complex beta
// (C), complex alpha (CS), window path (W: copy WC), element path (A)
#ifndef COSTA_MINB_8
#define COSTA_MINB_8 5
#endif
#ifndef COSTA_NBUF_8
#define COSTA_NBUF_8 1
#endif
#ifndef COSTA_MINB_8S
#define COSTA_MINB_8S 2
#endif
#ifndef COSTA_NBUF_8S
#define COSTA_NBUF_8S 3
#endif
#ifndef COSTA_MINB_8H
#define COSTA_MINB_8H 3
#endif
#ifndef COSTA_NBUF_8H
#define COSTA_NBUF_8H 2
#endif
#ifndef COSTA_MINB_8C
#define COSTA_MINB_8C 4
#endif
#ifndef COSTA_NBUF_8C
#define COSTA_NBUF_8C 1
#endif
#ifndef COSTA_MINB_8CS
#define COSTA_MINB_8CS 2
#endif
#ifndef COSTA_NBUF_8CS
#define COSTA_NBUF_8CS 3
#endif
#ifndef COSTA_MINB_8W
#define COSTA_MINB_8W COSTA_MINB_8
#endif
#ifndef COSTA_NBUF_8W
#define COSTA_NBUF_8W 2
#endif
#ifndef COSTA_NBUF_8WC
#define COSTA_NBUF_8WC 3
#endif
#ifndef COSTA_MINB_8A
#define COSTA_MINB_8A 4
#endif
// 16-byte: light kinds, scale, kinds that read A
#ifndef COSTA_MINB_16
#define COSTA_MINB_16 1
#endif
#ifndef COSTA_NBUF_16
#define COSTA_NBUF_16 2
#endif
#ifndef COSTA_MINB_16S
#define COSTA_MINB_16S 3
#endif
#ifndef COSTA_NBUF_16S
#define COSTA_NBUF_16S 1
#endif
#ifndef COSTA_MINB_16CS
#define COSTA_MINB_16CS 3
#endif
#ifndef COSTA_NBUF_16CS
#define COSTA_NBUF_16CS 1
#endif
#ifndef COSTA_MINB_16A
#define COSTA_MINB_16A 2
#endif
#ifndef COSTA_NBUF_16A
#define COSTA_NBUF_16A 1
#endif

struct Shape {
    int minb, nbuf;
};

// The table above.  es: element size; cplx: complex elements; mis: the
// misaligned-tile instance.
constexpr Shape launch_shape(int es, bool cplx, int kind, bool mis) {
    const bool reads_a = kind_reads_a(kind);
    if (es == 4) return reads_a ? Shape{COSTA_MINB_4A, COSTA_NBUF_4A} : Shape{COSTA_MINB_4, COSTA_NBUF_4};
    if (es == 16) {
        if (reads_a) return {COSTA_MINB_16A, COSTA_NBUF_16A};
        if (kind == K_CSCALE) return {COSTA_MINB_16CS, COSTA_NBUF_16CS};
        return kind == K_SCALE ? Shape{COSTA_MINB_16S, COSTA_NBUF_16S} : Shape{COSTA_MINB_16, COSTA_NBUF_16};
    }
    if (kind == K_CPLX) return {COSTA_MINB_8C, COSTA_NBUF_8C};
    if (kind == K_CSCALE) return {COSTA_MINB_8CS, COSTA_NBUF_8CS};
    if (kind == K_AXPBY) return {COSTA_MINB_8H, COSTA_NBUF_8H};
    if (mis) {
        if (reads_a) return {COSTA_MINB_8A, COSTA_NBUF_8};
        return {COSTA_MINB_8W, kind == K_COPY ? COSTA_NBUF_8WC : COSTA_NBUF_8W};
    }
    if (kind == K_SCALE && !cplx) return {COSTA_MINB_8S, COSTA_NBUF_8S};
    return {COSTA_MINB_8, COSTA_NBUF_8};
}

// Per element type: tile extent TS, 16-byte chunk width VEC (elements), and
// the lane mapping: CPR chunks cover one run of TS elements, a warp pass
// covers RPP runs, NPASS passes cover TS runs.  A staged tile is TS rows of
// CPR chunks (TS * TS elements); the element-wise path uses a TS x (TS + 1)
// array in the same buffer.
template <typename T> struct Cfg {
    static constexpr int TS = tile_extent(static_cast<int>(sizeof(T)));
    static constexpr int VEC = ET<T>::VEC;
    static constexpr int CPR = TS / VEC;
    static constexpr int RPP = 32 / CPR;
    static constexpr int NPASS = TS / RPP;
    static constexpr int PITCH = TS + 1;
    static constexpr int BUF_BYTES_RAW = TS * PITCH * static_cast<int>(sizeof(T));
    static constexpr int BUF_BYTES = (BUF_BYTES_RAW + 127) / 128 * 128;
    static constexpr int WARPS = sizeof(T) == 4 ? COSTA_WARPS_4 : COSTA_WARPS_8;
    // Lane maps give a run at most 32 lanes: a run's chunks (aligned path),
    // its elements (misaligned path of the kinds that read A) and one lane
    // per run or row (the window path's last pass) must each fit in a warp.
    // A larger tile extent would leave runs per pass at 0, and the copy
    // loops would never advance.
    static_assert(TS >= 1 && TS <= 32 && TS % VEC == 0, "tile extent must be a multiple of VEC in [VEC, 32]");
};

template <typename T, int KIND, bool MIS = false> struct KCfg {
    static constexpr bool HEAVY = KIND == K_AXPBY || KIND == K_CPLX || KIND == K_CSCALE;
    static constexpr bool READS_A = kind_reads_a(KIND);
    static constexpr int WARPS = Cfg<T>::WARPS;
    static constexpr Shape SHAPE = launch_shape(static_cast<int>(sizeof(T)), ET<T>::CPLX != 0, KIND, MIS);
    static constexpr int MINB = SHAPE.minb;
    static constexpr int NBUF = SHAPE.nbuf;
};

template <typename T> struct Chunk {
    union {
        uint4 raw;
        T e[ET<T>::VEC];
    };
};

// ---- asynchronous 16-byte global -> shared copies (sm_80+ cp.async) ----
__device__ __forceinline__ void cp_async16(void *smem, const void *gmem) {
    const unsigned s = static_cast<unsigned>(__cvta_generic_to_shared(smem));
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(s), "l"(gmem) : "memory");
}
// One element (4, 8 or 16 bytes) at its natural alignment.
template <int BYTES> __device__ __forceinline__ void cp_async_elem(void *smem, const void *gmem) {
    const unsigned s = static_cast<unsigned>(__cvta_generic_to_shared(smem));
    if constexpr (BYTES == 16)
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(s), "l"(gmem) : "memory");
    else
        asm volatile("cp.async.ca.shared.global [%0], [%1], %2;\n" ::"r"(s), "l"(gmem), "n"(BYTES) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N> __device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory");
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
    bool alpha_mid;      // both components of alpha zero or of magnitude in [2^-480, 2^480)
    bool scal_mid;       // the same for alpha and beta
    uint32_t conj_mask;  // 0x80000000 flips the sign of b's imaginary part (op = C)
    int32_t bexp;        // |beta| = 2^bexp (K_AXPBY2)
    uint32_t bsign_hi;   // sign bit of beta in a high word (K_AXPBY2)
    uint32_t p2_add;     // bexp << 20: exponent increment in a high word
    uint32_t p2_lo;      // admissible biased exponents: p2_lo + [0, p2_span]
    uint32_t p2_span;
};

// Combine of one element for a kind K_* (costa_internal.h); the kernel is
// compiled per kind.  b arrives conjugated (op = C) via conj_mask; for
// K_AXPBY2, a arrives already multiplied by beta (exactly, see prescale).
template <int KIND, typename R>
__device__ __forceinline__ R comb_real(R b, R a, const Sc &s) {
    if (KIND == K_COPY) return b;
    if (KIND == K_SCALE) return mulr(R(s.ar), b);
    if (KIND == K_AXPBY2) return fmar(R(s.ar), b, a);  // a arrives multiplied by beta
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

// Complex scalars: each component of alpha * b (+ beta * a) is the
// compensated dot product Dot2 of Ogita, Rump and Oishi ("Accurate sum and
// dot product", SIAM J. Sci. Comput. 26(6), 2005) over its 2 or 4 products,
// built on TwoProduct (one fma gives a product's rounding error exactly) and
// an error-free sum (two_sum below).  The result lies within u|x| + gamma_n^2 * sum|terms| of
// the exact component x (u the unit roundoff, n the number of terms): as if
// computed in twice the working precision and rounded once.  The running sum
// p is the plain sum of the rounded products; when it is not finite (an
// infinite or NaN input, an overflow) the error terms are undefined and p
// itself, the plain IEEE value, is the result.
__device__ __forceinline__ float addr(float a, float b) { return __fadd_rn(a, b); }
__device__ __forceinline__ double addr(double a, double b) { return __dadd_rn(a, b); }
__device__ __forceinline__ float subr(float a, float b) { return __fsub_rn(a, b); }
__device__ __forceinline__ double subr(double a, double b) { return __dsub_rn(a, b); }

// p + h = t + q exactly.  Float: Knuth's TwoSum (6 operations).  Double:
// the two operands ordered by exponent on the integer pipes (their high
// words without the sign), then Dekker's Fast2Sum (3 operations), which is
// exact when the first operand's exponent is not below the second's: the
// same t and q, with half the FP64 operations, the pipe that bounds the
// complex kinds of c128 on GB300.
__device__ __forceinline__ void two_sum(float p, float h, float &t, float &q) {
    t = addr(p, h);
    const float z = subr(t, p);
    q = addr(subr(p, subr(t, z)), subr(h, z));
}
__device__ __forceinline__ void two_sum(double p, double h, double &t, double &q) {
    const unsigned ep = static_cast<unsigned>(__double2hiint(p)) & 0x7FFFFFFFu;
    const unsigned eh = static_cast<unsigned>(__double2hiint(h)) & 0x7FFFFFFFu;
    const double a = eh > ep ? h : p, b = eh > ep ? p : h;  // exponent of a >= exponent of b
    t = addr(a, b);
    q = subr(b, subr(t, a));
}

template <typename R> struct Dot2 {
    R p, s;  // running sum of the rounded products; sum of the error terms
    __device__ __forceinline__ Dot2(R x, R y) {
        p = mulr(x, y);
        s = fmar(x, y, -p);
    }
    __device__ __forceinline__ void add(R x, R y) {
        const R h = mulr(x, y);
        const R r = fmar(x, y, -h);  // x * y = h + r exactly
        R t, q;
        two_sum(p, h, t, q);
        p = t;
        s = addr(s, addr(q, r));
    }
    __device__ __forceinline__ R result() const { return isfinite(p) ? addr(p, s) : p; }
};

// A double that is zero or of magnitude in [2^-480, 2^480): products of two
// such values neither overflow nor lose their rounding error to underflow.
__device__ __forceinline__ bool mid_range(double v) {
    const unsigned hi = static_cast<unsigned>(__double2hiint(v));
    const unsigned lo = static_cast<unsigned>(__double2loint(v));
    const unsigned e = (hi >> 20) & 0x7FFu;
    return (((hi & 0x7FFFFFFFu) | lo) == 0u) || (e - (1023u - 480u)) < 960u;
}

// x * y + sgn * (z * t) with Kahan's algorithm for 2 x 2 determinants: w =
// z * t rounded, its error e exactly by one fma, then (x * y + sgn * w)
// rounded by a second fma and sgn * e added.  Jeannerod, Louvet and Muller
// ("Further analysis of Kahan's algorithm for the accurate computation of
// 2 x 2 determinants", Math. Comp. 82, 2013) bound its error by 2u|exact|
// when nothing overflows or underflows: within 2 ulps of the exact value,
// and so of the oracle's compensated result.  4 FP64 operations instead of
// Dot2's 13.
__device__ __forceinline__ double kahan2(double x, double y, double z, double t, bool minus) {
    const double w = __dmul_rn(z, t);
    const double e = __fma_rn(z, t, -w);  // z * t = w + e exactly
    return minus ? __dsub_rn(__fma_rn(x, y, -w), e) : __dadd_rn(__fma_rn(x, y, w), e);
}

// Passes of a tile that the drain of double complex data with complex
// scalars evaluates together (stage_drain).
#ifndef COSTA_FX_GROUP
#define COSTA_FX_GROUP 2
#endif
// Passes that the drain of double complex data with a complex alpha and
// beta = 0 evaluates together: the last in fixed point, the others by
// Kahan's algorithm (0: every pass by Kahan's algorithm, one at a time).
#ifndef COSTA_FX_CS_PERIOD
#define COSTA_FX_CS_PERIOD 2
#endif

// Every operand of a double complex alpha * b + beta * a in the middle range
// (b as it enters the combine, after any conjugation).
__device__ __forceinline__ bool cplx_mid(const double2 &b, const double2 &a, const Sc &s) {
    return s.scal_mid && mid_range(b.x) && mid_range(b.y) && mid_range(a.x) && mid_range(a.y);
}
template <typename C> __device__ __forceinline__ bool cplx_mid(const C &, const C &, const Sc &) {
    return false;
}

// alpha * b + beta * a for double complex data and complex scalars, each
// component the sum of its four products in fixed point on the integer pipes
// (fxdot.h): within 0.5 ulp of the component plus 2^-5 ulp of its largest
// product, with no FP64 operation.  Dot2 takes 24 FP64 operations per
// component, and the FP64 pipe is narrow on GB300.  Every operand must be in
// the middle range (cplx_mid).
__device__ __forceinline__ double2 fx_cplx(const double2 &b, const double2 &a, const Sc &s) {
    const fx::Op fbx = fx::unpack(b.x), fby = fx::unpack(b.y), fax = fx::unpack(a.x), fay = fx::unpack(a.y);
    const fx::Op far = fx::unpack(s.ar), fai = fx::unpack(s.ai), fbr = fx::unpack(s.br), fbi = fx::unpack(s.bi);
    // ar bx - ai by + br ax - bi ay;  ar by + ai bx + br ay + bi ax
    const fx::Term re[4] = {fx::mul(far, fbx, 0u), fx::mul(fai, fby, 1u), fx::mul(fbr, fax, 0u),
                            fx::mul(fbi, fay, 1u)};
    const fx::Term im[4] = {fx::mul(far, fby, 0u), fx::mul(fai, fbx, 0u), fx::mul(fbr, fay, 0u),
                            fx::mul(fbi, fax, 0u)};
    double2 o;
    o.x = fx::sum(re);
    o.y = fx::sum(im);
    return o;
}

// alpha * b for double complex data and a complex alpha, each component the
// sum of its two products in fixed point on the integer pipes (fxdot.h).
// Every operand must be in the middle range.
__device__ __forceinline__ double2 fx_cscale(const double2 &b, const Sc &s) {
    const fx::Op fbx = fx::unpack(b.x), fby = fx::unpack(b.y);
    const fx::Op far = fx::unpack(s.ar), fai = fx::unpack(s.ai);
    const fx::Term re[2] = {fx::mul(far, fbx, 0u), fx::mul(fai, fby, 1u)};  // ar bx - ai by
    const fx::Term im[2] = {fx::mul(far, fby, 0u), fx::mul(fai, fbx, 0u)};  // ar by + ai bx
    double2 o;
    o.x = fx::sum(re);
    o.y = fx::sum(im);
    return o;
}

template <int KIND, typename C, typename R>
__device__ __forceinline__ C combine_c(C b, C a, const Sc &s) {
    b.y = flip_sign(b.y, s.conj_mask);
    C o;
    if (KIND != K_CPLX && KIND != K_CSCALE) {
        o.x = comb_real<KIND, R>(b.x, a.x, s);
        o.y = comb_real<KIND, R>(b.y, a.y, s);
        return o;
    }
    if constexpr (KIND == K_CSCALE && sizeof(R) == 8) {
        // the FP64 pipe is this kind's limit: two-term components take
        // Kahan's algorithm when every operand is in the middle range (the
        // others, and all non-finite values, take Dot2 below)
        if (s.alpha_mid && mid_range(b.x) && mid_range(b.y)) {
            o.x = kahan2(s.ar, b.x, s.ai, b.y, true);   // ar bx - ai by
            o.y = kahan2(s.ar, b.y, s.ai, b.x, false);  // ar by + ai bx
            return o;
        }
    }
    if constexpr (KIND == K_CPLX && sizeof(R) == 8) {
        // four-term components: in fixed point on the integer pipes when
        // every operand is in the middle range (fx_cplx)
        if (cplx_mid(b, a, s)) return fx_cplx(b, a, s);
    }
    const R ar = R(s.ar), ai = R(s.ai);
    Dot2<R> re(ar, b.x), im(ar, b.y);
    re.add(-ai, b.y);
    im.add(ai, b.x);
    if (KIND == K_CPLX) {
        const R br = R(s.br), bi = R(s.bi);
        re.add(br, a.x);
        re.add(-bi, a.y);
        im.add(br, a.y);
        im.add(bi, a.x);
    }
    o.x = re.result();
    o.y = im.result();
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
// The source's runs (its contiguous axis) are rows of the staged tile: for a
// copy tile row y holds x = 0..nx-1, for a transposed tile row x holds
// y = 0..ny-1.
template <typename T> struct Geom {
    T *dst;
    const T *src;
    int64_t dld, sld;
    int nx, ny;
    int prob;
    bool transpose, fast, conj, elem;
};

// Chunk c of staged row r lives in slot c ^ swz(r): across the VEC rows that
// one output chunk reads, and across neighbouring chunks, the slots differ,
// so a transposed read needs only the minimum number of wavefronts.
template <typename T>
__device__ __forceinline__ int swz(int r) { return (r / Cfg<T>::VEC) & 7; }

template <typename T>
__device__ __forceinline__ unsigned char *slot(unsigned char *buf, int r, int c) {
    return buf + (r * Cfg<T>::CPR + (c ^ swz<T>(r))) * 16;
}

// Lane mapping for runs of `chunks` 16-byte chunks (1 <= chunks <= CPR):
// lpr = the next power of two >= chunks lanes per run, 32 / lpr runs per warp
// pass.  Narrow tiles thus keep all lanes busy instead of leaving the lanes
// beyond the run idle.
struct LaneMap {
    int c;    // chunk of this lane within its run
    int r0;   // run of this lane in pass 0
    int rpp;  // runs per pass
};
__device__ __forceinline__ LaneMap lane_map(int chunks, int lane) {
    const int sh = chunks <= 1 ? 0 : 32 - __clz(chunks - 1);
    LaneMap m;
    m.c = lane & ((1 << sh) - 1);
    m.r0 = lane >> sh;
    m.rpp = 32 >> sh;
    return m;
}

// Issue the cp.async copies of a fast tile's source into `buf`.
template <typename T>
__device__ __forceinline__ void stage_issue(const Geom<T> &g, unsigned char *buf, int lane) {
    using C = Cfg<T>;
    const int runs = g.transpose ? g.nx : g.ny;               // source runs
    const int chunks = (g.transpose ? g.ny : g.nx) / C::VEC;  // chunks per run
    const LaneMap m = lane_map(chunks, lane);
    if (m.c >= chunks) return;
#pragma unroll 4
    for (int r = m.r0; r < runs; r += m.rpp)
        cp_async16(slot<T>(buf, r, m.c), g.src + static_cast<int64_t>(r) * g.sld + m.c * C::VEC);
}

// beta * a for beta = +-2^k without the FP64 pipe.  For a zero or a normal a
// whose biased exponent e stays in [1, 2046] after adding k, the product is
// exact: a's high word with k added to the exponent field (zeros unchanged)
// and the sign flipped for negative beta.  Sc holds the admissible exponent
// range as p2_lo + [0, p2_span].  `bad` collects the other cases
// (subnormals, infinities, NaNs, products leaving the normal range), which
// the multiply handles.
__device__ __forceinline__ bool pow2_bad(double a, const Sc &s) {
    const unsigned hi = static_cast<unsigned>(__double2hiint(a));
    const unsigned lo = static_cast<unsigned>(__double2loint(a));
    const unsigned e = (hi >> 20) & 0x7FFu;
    const bool zero = ((hi & 0x7FFFFFFFu) | lo) == 0u;
    return !zero && (e - s.p2_lo) > s.p2_span;
}
__device__ __forceinline__ double pow2_apply(double a, const Sc &s) {
    const unsigned hi = static_cast<unsigned>(__double2hiint(a));
    const unsigned lo = static_cast<unsigned>(__double2loint(a));
    const unsigned nh = (hi & 0x7FF00000u) ? hi + s.p2_add : hi;  // zeros keep their exponent
    return __hiloint2double(static_cast<int>(nh ^ s.bsign_hi), static_cast<int>(lo));
}

// Scales the loaded A chunks (the first `npass` passes) by beta in place for
// kind K_AXPBY2.  Double data takes the exact integer path unless some lane
// of the warp holds a value it does not cover; that choice is one warp vote,
// so the scarce FP64 pipe never runs predicated-off multiplies.  beta = +-1
// needs at most a sign flip.  Float data multiplies (the FP32 pipe is wide).
template <typename T, int N>
__device__ __forceinline__ void prescale(Chunk<T> (&av)[N], int npass, const Sc &s) {
    using R = typename ET<T>::R;
    constexpr int PER = 16 / static_cast<int>(sizeof(R));  // reals per chunk
    if constexpr (sizeof(R) == 8) {
        if (s.bexp == 0) {
            if (s.bsign_hi) {
#pragma unroll
                for (int p = 0; p < N; ++p) {
                    if (p >= npass) break;
                    av[p].raw.y ^= s.bsign_hi;
                    av[p].raw.w ^= s.bsign_hi;
                }
            }
            return;
        }
        bool bad = false;
#pragma unroll
        for (int p = 0; p < N; ++p) {
            if (p >= npass) break;
            const double *v = reinterpret_cast<const double *>(&av[p]);
#pragma unroll
            for (int k = 0; k < PER; ++k) bad |= pow2_bad(v[k], s);
        }
        if (__any_sync(0xffffffffu, bad)) {
#pragma unroll
            for (int p = 0; p < N; ++p) {
                if (p >= npass) break;
                double *v = reinterpret_cast<double *>(&av[p]);
#pragma unroll
                for (int k = 0; k < PER; ++k) v[k] = __dmul_rn(s.br, v[k]);
            }
        } else {
#pragma unroll
            for (int p = 0; p < N; ++p) {
                if (p >= npass) break;
                double *v = reinterpret_cast<double *>(&av[p]);
#pragma unroll
                for (int k = 0; k < PER; ++k) v[k] = pow2_apply(v[k], s);
            }
        }
    } else {
#pragma unroll
        for (int p = 0; p < N; ++p) {
            if (p >= npass) break;
            float *v = reinterpret_cast<float *>(&av[p]);
#pragma unroll
            for (int k = 0; k < PER; ++k) v[k] = __fmul_rn(float(s.br), v[k]);
        }
    }
}

// Loads the tile's A chunks (kinds that read A) in the drain's lane mapping.
// Called by all 32 lanes (prescale votes).
template <typename T, int KIND>
__device__ __forceinline__ void load_a(const Geom<T> &g, const Sc &s, Chunk<T> (&av)[Cfg<T>::NPASS],
                                       int lane) {
    using C = Cfg<T>;
    if (!kind_reads_a(KIND)) return;
    const int chunks = g.nx / C::VEC;
    const LaneMap m = lane_map(chunks, lane);
    const int x0 = m.c * C::VEC;
    const bool on = m.c < chunks;
    const int npass = (g.ny + m.rpp - 1) / m.rpp;
#pragma unroll
    for (int p = 0; p < C::NPASS; ++p) {
        if (p >= npass) break;  // uniform across the warp
        const int y = p * m.rpp + m.r0;
        av[p].raw = make_uint4(0, 0, 0, 0);
        if (on && y < g.ny) av[p] = load_rw(g.dst + static_cast<int64_t>(y) * g.dld + x0);
    }
    if (KIND == K_AXPBY2) prescale<T>(av, npass, s);
}

// ---- TMA staging layout (the f64 general-beta kind; every kind with COSTA_TMA=1; see tma.cpp) ----
// A TMA-staged tile is boxes of 16 runs x 128 bytes: box (br, bl) (run / 16,
// byte along the run / 128) at (br * TBL + bl) * 2048 bytes, 1024-byte
// aligned, each a stack of 128-byte rows whose 16-byte chunks the TMA unit
// swizzles (128-byte mode): chunk j of row r lands at j ^ (r mod 8).
template <typename T> struct TCfg {
    static constexpr int TBL = Cfg<T>::TS * static_cast<int>(sizeof(T)) / 128;  // boxes along a run
    static constexpr int BUF = 2 * TBL * 2048;                                    // up to 32 runs
    static_assert(Cfg<T>::TS * sizeof(T) % 128 == 0, "a full run is whole boxes");
};
template <typename T>
__device__ __forceinline__ unsigned char *slot_t(unsigned char *buf, int r, int c) {
    return buf + ((r >> 4) * TCfg<T>::TBL + (c >> 3)) * 2048 + (r & 15) * 128 + (((c & 7) ^ (r & 7)) << 4);
}
// Chunk c of staged run r in the cp.async layout (TL = false) or the TMA one.
template <typename T, bool TL>
__device__ __forceinline__ unsigned char *slot_any(unsigned char *buf, int r, int c) {
    if constexpr (TL) return slot_t<T>(buf, r, c);
    else return slot<T>(buf, r, c);
}

// The drain of double complex data with a complex beta loads A itself, a
// few passes ahead (stage_drain); for the other kinds that read A the
// caller loads the tile's A chunks into registers first (load_a).
template <typename T, int KIND> __host__ __device__ constexpr bool drain_loads_a() {
    return KIND == K_CPLX && sizeof(T) == 16;
}

// Write a staged fast tile to A, combining with A when the kind reads it.
template <typename T, int KIND, bool TL = false>
__device__ __forceinline__ void stage_drain(const Geom<T> &g, const Sc &s, unsigned char *buf,
                                            const Chunk<T> (&av)[Cfg<T>::NPASS], int lane) {
    using C = Cfg<T>;
    const int chunks = g.nx / C::VEC;
    const LaneMap m = lane_map(chunks, lane);
    if (m.c >= chunks) return;
    const int x0 = m.c * C::VEC;
    const int npass = (g.ny + m.rpp - 1) / m.rpp;
    if constexpr ((KIND == K_CPLX || (KIND == K_CSCALE && COSTA_FX_CS_PERIOD > 0)) && sizeof(T) == 16) {
        // double complex with complex scalars: G passes at a time in
        // straight-line code, so that their evaluations overlap.  Four-term
        // components (complex beta) are all summed in fixed point on the
        // integer pipes (about 150 instructions each, in long dependent
        // chains); two-term ones (complex alpha, beta = 0) split the passes
        // between Kahan's algorithm on the FP64 pipe and the fixed-point sum,
        // so that both pipes work.  The loop stays rolled: unrolled over the
        // tile's passes, the fixed-point sums made a body of about 14,000
        // instructions, and instruction fetch stalled the warps.  So A is
        // not held as a whole tile in registers (av is unused here; the
        // callers do not load it for this kind): each iteration loads the A
        // chunks of the group two ahead of the one it combines.
        constexpr int G = KIND == K_CPLX ? COSTA_FX_GROUP : COSTA_FX_CS_PERIOD;
        T a_next[2][G];
        auto load_group = [&](int q0, T (&dst)[G]) {
#pragma unroll
            for (int j = 0; j < G; ++j) {
                const int y = (q0 + j) * m.rpp + m.r0;
                dst[j] = T{0.0, 0.0};
                if (KIND == K_CPLX && q0 + j < npass && y < g.ny)
                    dst[j] = load_rw(g.dst + static_cast<int64_t>(y) * g.dld + x0).e[0];
            }
        };
        load_group(0, a_next[0]);
        load_group(G, a_next[1]);
#pragma unroll 1
        for (int p0 = 0; p0 < npass; p0 += G) {
            T bb[G], aa[G];
#pragma unroll
            for (int j = 0; j < G; ++j) {
                aa[j] = a_next[0][j];
                a_next[0][j] = a_next[1][j];
            }
            load_group(p0 + 2 * G, a_next[1]);
            bool ok[G];
#pragma unroll
            for (int j = 0; j < G; ++j) {
                const int y = (p0 + j) * m.rpp + m.r0;
                ok[j] = p0 + j < npass && y < g.ny;
                bb[j] = ok[j] ? *reinterpret_cast<const T *>(slot_any<T, TL>(buf, g.transpose ? x0 : y,
                                                                            g.transpose ? y : m.c))
                              : T{0.0, 0.0};
                bb[j].y = flip_sign(bb[j].y, s.conj_mask);
            }
            bool mid = KIND == K_CPLX || s.alpha_mid;
#pragma unroll
            for (int j = 0; j < G; ++j)
                mid = mid && (KIND == K_CPLX ? cplx_mid(bb[j], aa[j], s) : mid_range(bb[j].x) && mid_range(bb[j].y));
            T o[G];
            if (mid) {
#pragma unroll
                for (int j = 0; j < G; ++j) {
                    if (KIND == K_CPLX) {
                        o[j] = fx_cplx(bb[j], aa[j], s);
                    } else if (j == G - 1) {
                        o[j] = fx_cscale(bb[j], s);
                    } else {
                        o[j].x = kahan2(s.ar, bb[j].x, s.ai, bb[j].y, true);   // ar bx - ai by
                        o[j].y = kahan2(s.ar, bb[j].y, s.ai, bb[j].x, false);  // ar by + ai bx
                    }
                }
            } else {
#pragma unroll
                for (int j = 0; j < G; ++j) {
                    bb[j].y = flip_sign(bb[j].y, s.conj_mask);  // combine conjugates again
                    o[j] = combine<KIND>(bb[j], aa[j], s);
                }
            }
#pragma unroll
            for (int j = 0; j < G; ++j)
                if (ok[j]) *(g.dst + static_cast<int64_t>((p0 + j) * m.rpp + m.r0) * g.dld + x0) = o[j];
        }
        return;
    }
#pragma unroll
    for (int p = 0; p < C::NPASS; ++p) {
        if (p >= npass) break;  // uniform across the warp
        const int y = p * m.rpp + m.r0;
        if (y < g.ny) {
            Chunk<T> b;
            if (g.transpose) {
                // element (x0 + e, y) sits in row x0 + e, chunk y / VEC, lane y % VEC
                const int cy = y / C::VEC, ey = y % C::VEC;
#pragma unroll
                for (int e = 0; e < C::VEC; ++e)
                    b.e[e] = reinterpret_cast<const T *>(slot_any<T, TL>(buf, x0 + e, cy))[ey];
            } else {
                b.raw = *reinterpret_cast<const uint4 *>(slot_any<T, TL>(buf, y, m.c));
            }
            Chunk<T> o;
#pragma unroll
            for (int e = 0; e < C::VEC; ++e) o.e[e] = combine<KIND>(b.e[e], av[p].e[e], s);
            store(g.dst + static_cast<int64_t>(y) * g.dld + x0, o);
        }
    }
}

// K_AXPBY2 takes a multiplied by beta (a power of two: exact); other kinds
// take a as it is.
template <int KIND> __device__ __forceinline__ float premul(float a, const Sc &s) {
    return KIND == K_AXPBY2 ? __fmul_rn(float(s.br), a) : a;
}
template <int KIND> __device__ __forceinline__ double premul(double a, const Sc &s) {
    return KIND == K_AXPBY2 ? __dmul_rn(s.br, a) : a;
}
template <int KIND> __device__ __forceinline__ float2 premul(float2 a, const Sc &s) {
    return KIND == K_AXPBY2 ? make_float2(__fmul_rn(float(s.br), a.x), __fmul_rn(float(s.br), a.y)) : a;
}
template <int KIND> __device__ __forceinline__ double2 premul(double2 a, const Sc &s) {
    return KIND == K_AXPBY2 ? make_double2(__dmul_rn(s.br, a.x), __dmul_rn(s.br, a.y)) : a;
}

// Element-wise fallback of the aligned kernel for a tile that is not on the
// vector path (the host lists none there; misaligned tiles go to the
// one-element-per-lane instance): lanes strided along the contiguous axis of
// each phase, through a TS x (TS + 1) array in `buf`.
template <typename T, int KIND>
__device__ __forceinline__ void tile_general(const Geom<T> &g, const Sc &s, unsigned char *buf, int lane) {
    using C = Cfg<T>;
    constexpr bool READ_A = kind_reads_a(KIND);
    T *sm = reinterpret_cast<T *>(buf);
    const int n = g.nx * g.ny;
    if (!g.transpose) {
        for (int k = lane; k < n; k += 32) {
            const int y = k / g.nx, x = k - y * g.nx;
            T *d = g.dst + static_cast<int64_t>(y) * g.dld + x;
            const T a = READ_A ? premul<KIND>(*d, s) : T();
            *d = combine<KIND>(__ldg(g.src + static_cast<int64_t>(y) * g.sld + x), a, s);
        }
        return;
    }
    for (int k = lane; k < n; k += 32) {
        const int x = k / g.ny, y = k - x * g.ny;
        sm[y * C::PITCH + x] = __ldg(g.src + static_cast<int64_t>(x) * g.sld + y);
    }
    __syncwarp();
    for (int k = lane; k < n; k += 32) {
        const int y = k / g.nx, x = k - y * g.nx;
        T *d = g.dst + static_cast<int64_t>(y) * g.dld + x;
        const T a = READ_A ? premul<KIND>(*d, s) : T();
        *d = combine<KIND>(sm[y * C::PITCH + x], a, s);
    }
}

// ---- misaligned tiles ----
//
// A tile whose runs do not start on 16-byte boundaries (an odd leading
// dimension, a block at an odd offset) or whose extents are not whole chunks
// takes one of two paths (measured on GB300: each is the faster one where
// it is used).
//  - Kinds that do not read A move 16-byte chunks over each run's window
//    (the aligned chunks that cover the run), like an aligned tile; 4-byte
//    tiles whose target runs are misaligned (flag TF_ELEM, set by the host)
//    take the element path instead.
//  - Kinds that read A move one element per lane.
// The window path stages into the TS x CPR swizzled slots of an aligned
// tile's buffer plus one extra column of TS chunks, the element path into
// TS x TS elements of the same buffer.

// ---- 16-byte windows (kinds that do not read A) ----
//
// A run of len elements at phase ph (its start address mod 16, in elements)
// has ceil((ph + len) / VEC) window chunks, at most CPR + 1.
//  - Source: every window chunk is copied whole.  The bytes beyond the run
//    lie in the same aligned 16-byte chunk as bytes of the run (so on the
//    same page of the same allocation) and are only read, never used.
//  - A: a window chunk wholly inside the run is stored with one 16-byte
//    access; a chunk that the run covers in part (the first and the last of a
//    run) is stored element by element, so nothing outside the tile is
//    written.
// The staged run keeps its phase: element c of source run r sits at window
// position ph_r + c.  Window chunk k < CPR lives in slot k of staged row r;
// chunk CPR in the extra column.
//
// Lanes take the window chunks k < CPR with the aligned tile's lane map, and
// chunk CPR of every run in one more pass.  A lane's runs are a multiple of
// VEC apart (runs per pass = 32 / lanes per run >= 32 / CPR = VEC, both
// powers of two), so they share their phase: the lane's chunk covers the same
// tile columns in all its passes and, transposed, reads the same staged rows.

template <typename T> struct WCfg {
    static constexpr int XCOL = Cfg<T>::TS * Cfg<T>::CPR * 16;  // byte offset of the extra column
    static constexpr int BUF_BYTES = (XCOL + Cfg<T>::TS * 16 + 127) / 128 * 128;
};

// Staged element at window position q of run r.
template <typename T>
__device__ __forceinline__ const T &welem(unsigned char *buf, int r, int q) {
    using C = Cfg<T>;
    const int j = q / C::VEC;
    const unsigned char *c = j < C::CPR ? slot<T>(buf, r, j) : buf + WCfg<T>::XCOL + r * 16;
    return reinterpret_cast<const T *>(c)[q % C::VEC];
}

// Phase (start address mod 16, in elements) of run r of a surface whose run
// 0 starts at p and whose runs are ld elements apart.
template <typename T>
__device__ __forceinline__ int phase(const T *p, int64_t ld, int r) {
    constexpr int V = Cfg<T>::VEC;
    const int p0 = static_cast<int>((reinterpret_cast<uintptr_t>(p) & 15u) / sizeof(T));
    return (p0 + r * static_cast<int>(ld & (V - 1))) & (V - 1);
}

// Window chunks per run of len elements (the most any phase needs), and
// those of them below CPR.
template <typename T> __device__ __forceinline__ int wchunks(int len) {
    return (len + 2 * Cfg<T>::VEC - 2) / Cfg<T>::VEC;
}
template <typename T> __device__ __forceinline__ int wmain(int len) { return min(Cfg<T>::CPR, wchunks<T>(len)); }

template <typename T>
__device__ __forceinline__ void stage_issue_w(const Geom<T> &g, unsigned char *buf, int lane) {
    using C = Cfg<T>;
    const int runs = g.transpose ? g.nx : g.ny;
    const int len = g.transpose ? g.ny : g.nx;  // elements per run
    const int cm = wmain<T>(len);
    const LaneMap m = lane_map(cm, lane);
    const int ph = phase<T>(g.src, g.sld, m.r0);  // the phase of all this lane's runs
    if (m.c < cm && m.c * C::VEC < ph + len) {
        const T *s0 = g.src - ph + m.c * C::VEC;
#pragma unroll 4
        for (int r = m.r0; r < runs; r += m.rpp)
            cp_async16(slot<T>(buf, r, m.c), s0 + static_cast<int64_t>(r) * g.sld);
    }
    if (wchunks<T>(len) > C::CPR && lane < runs) {  // chunk CPR: lane = run
        const int pr = phase<T>(g.src, g.sld, lane);
        if (C::CPR * C::VEC < pr + len)
            cp_async16(buf + WCfg<T>::XCOL + lane * 16,
                       g.src + static_cast<int64_t>(lane) * g.sld - pr + C::CPR * C::VEC);
    }
}

// The staged elements of tile columns x0 .. x0 + VEC - 1 of tile row y
// (columns outside [0, nx) read an in-tile element; they are not stored).
template <typename T>
__device__ __forceinline__ Chunk<T> staged_window(const Geom<T> &g, unsigned char *buf, int x0, int y) {
    using C = Cfg<T>;
    Chunk<T> b;
    if (g.transpose) {
#pragma unroll
        for (int i = 0; i < C::VEC; ++i) {
            const int x = min(max(x0 + i, 0), g.nx - 1);  // source run x, position y
            b.e[i] = welem<T>(buf, x, phase<T>(g.src, g.sld, x) + y);
        }
    } else {
        const int ph = phase<T>(g.src, g.sld, y);  // source run y, positions x
#pragma unroll
        for (int i = 0; i < C::VEC; ++i) b.e[i] = welem<T>(buf, y, ph + min(max(x0 + i, 0), g.nx - 1));
    }
    return b;
}

// Writes the tile columns of x0 .. x0 + VEC - 1 (a window chunk of tile row
// y) that lie in [0, nx), element by element.
template <typename T, int KIND>
__device__ __forceinline__ void drain_partial_w(const Geom<T> &g, const Sc &s, unsigned char *buf, int x0, int y) {
    using C = Cfg<T>;
    const Chunk<T> b = staged_window<T>(g, buf, x0, y);
    T *row = g.dst + static_cast<int64_t>(y) * g.dld;
#pragma unroll
    for (int i = 0; i < C::VEC; ++i)
        if (x0 + i >= 0 && x0 + i < g.nx) row[x0 + i] = combine<KIND>(b.e[i], T(), s);
}

// The full window chunks of one lane: tile columns x0 .. x0 + VEC - 1 (all
// inside the tile) of rows r0, r0 + rpp, ...  rpp is a multiple of VEC, so
// every staged run the lane reads keeps its phase and its offset within a
// chunk from pass to pass: they are computed once, and a pass advances the
// staged chunk index only.
template <typename T, int KIND>
__device__ __forceinline__ void drain_full_w(const Geom<T> &g, const Sc &s, unsigned char *buf, int x0, int r0,
                                             int rpp) {
    using C = Cfg<T>;
    constexpr int V = C::VEC, ES = static_cast<int>(sizeof(T)), ROW = C::CPR * 16;
    T *d = g.dst + static_cast<int64_t>(r0) * g.dld + x0;
    const int64_t dstep = static_cast<int64_t>(rpp) * g.dld;
    if (g.transpose) {
        // element (x0 + e, y): staged run x0 + e, window position ph + y
        const int dj = rpp / V;
        int j0[V], sw[V], off[V], xo[V];
#pragma unroll
        for (int e = 0; e < V; ++e) {
            const int x = x0 + e, q = phase<T>(g.src, g.sld, x) + r0;
            j0[e] = q / V;
            sw[e] = swz<T>(x);
            off[e] = x * ROW + (q % V) * ES;
            xo[e] = WCfg<T>::XCOL + x * 16 + (q % V) * ES;
        }
#pragma unroll 4
        for (int p = 0, y = r0; y < g.ny; ++p, y += rpp) {
            Chunk<T> b, o;
#pragma unroll
            for (int e = 0; e < V; ++e) {
                const int j = j0[e] + p * dj;
                b.e[e] = *reinterpret_cast<const T *>(buf + (j < C::CPR ? off[e] + ((j ^ sw[e]) << 4) : xo[e]));
            }
#pragma unroll
            for (int e = 0; e < V; ++e) o.e[e] = combine<KIND>(b.e[e], T(), s);
            store(d, o);
            d += dstep;
        }
    } else {
        // row y: staged run y, window positions q .. q + VEC - 1 (chunk j
        // from element w, then chunk j + 1)
        const int q = phase<T>(g.src, g.sld, r0) + x0, j = q / V, w = q % V;
#pragma unroll 4
        for (int y = r0; y < g.ny; y += rpp) {
            const int sw = swz<T>(y);
            const int o0 = j < C::CPR ? y * ROW + ((j ^ sw) << 4) : WCfg<T>::XCOL + y * 16;
            const int o1 = j + 1 < C::CPR ? y * ROW + (((j + 1) ^ sw) << 4) : WCfg<T>::XCOL + y * 16;
            Chunk<T> b, o;
#pragma unroll
            for (int e = 0; e < V; ++e) {
                const int k = w + e;
                b.e[e] = *reinterpret_cast<const T *>(buf + (k < V ? o0 + k * ES : o1 + (k - V) * ES));
            }
#pragma unroll
            for (int e = 0; e < V; ++e) o.e[e] = combine<KIND>(b.e[e], T(), s);
            store(d, o);
            d += dstep;
        }
    }
}

// Full window chunks go out in the lane-map passes, with 16-byte stores
// only; the partial ones (a run's first chunk when its phase is not 0, its
// last when the run does not fill it) in one more pass, lane = tile row.
template <typename T, int KIND>
__device__ __forceinline__ void stage_drain_w(const Geom<T> &g, const Sc &s, unsigned char *buf, int lane) {
    using C = Cfg<T>;
    static_assert(!kind_reads_a(KIND), "the window path does not read A");
    const int cm = wmain<T>(g.nx);
    const LaneMap m = lane_map(cm, lane);
    const int x0 = m.c * C::VEC - phase<T>(g.dst, g.dld, m.r0);  // first tile column of the lane's chunk
    if (m.c < cm && x0 >= 0 && x0 + C::VEC <= g.nx) {
        drain_full_w<T, KIND>(g, s, buf, x0, m.r0, m.rpp);
    }
    if (lane < g.ny) {
        const int ph = phase<T>(g.dst, g.dld, lane);
        const int last = (ph + g.nx - 1) / C::VEC;  // last window chunk of the row
        const int xl = last * C::VEC - ph;
        if (ph > 0) drain_partial_w<T, KIND>(g, s, buf, -ph, lane);
        if (xl + C::VEC > g.nx && (last > 0 || ph == 0)) drain_partial_w<T, KIND>(g, s, buf, xl, lane);
    }
}

// ---- one element per lane (kinds that read A) ----
//
// cp.async of single elements into shared memory, A's elements loaded into
// registers before the wait, and element-wide, still coalesced, stores.
// Staged rows are TS elements wide; element c of row r lives at position
// c ^ (r mod TS), so that lanes reading one position across consecutive rows
// (the transposed read) hit distinct banks.

template <typename T>
__device__ __forceinline__ T *slot_e(unsigned char *buf, int r, int c) {
    using C = Cfg<T>;
    return reinterpret_cast<T *>(buf) + r * C::TS + (c ^ (r & (C::TS - 1)));
}

template <typename T>
__device__ __forceinline__ void stage_issue_e(const Geom<T> &g, unsigned char *buf, int lane) {
    const int runs = g.transpose ? g.nx : g.ny;
    const int len = g.transpose ? g.ny : g.nx;  // elements per run
    const LaneMap m = lane_map(len, lane);
    if (m.c >= len) return;
#pragma unroll 4
    for (int r = m.r0; r < runs; r += m.rpp)
        cp_async_elem<sizeof(T)>(slot_e<T>(buf, r, m.c), g.src + static_cast<int64_t>(r) * g.sld + m.c);
}

// Element e of the warp's NPASS * VEC register elements (compile-time e).
template <typename T> __device__ __forceinline__ T &elem(Chunk<T> (&av)[Cfg<T>::NPASS], int e) {
    return av[e / Cfg<T>::VEC].e[e % Cfg<T>::VEC];
}

template <typename T, int KIND>
__device__ __forceinline__ void load_a_e(const Geom<T> &g, const Sc &s, Chunk<T> (&av)[Cfg<T>::NPASS], int lane) {
    using C = Cfg<T>;
    if (!kind_reads_a(KIND)) return;
    constexpr int NE = C::NPASS * C::VEC;  // elements per lane, full tile
    const LaneMap m = lane_map(g.nx, lane);
    const bool on = m.c < g.nx;
    const int npass = (g.ny + m.rpp - 1) / m.rpp;
    const int npad = (npass + C::VEC - 1) / C::VEC * C::VEC;  // whole chunks for prescale
#pragma unroll
    for (int p = 0; p < NE; ++p) {
        if (p >= npad) break;  // uniform across the warp
        const int y = p * m.rpp + m.r0;
        T a;
        if constexpr (ET<T>::CPLX) a = T{0, 0}; else a = T(0);
        if (on && p < npass && y < g.ny) a = g.dst[static_cast<int64_t>(y) * g.dld + m.c];
        elem<T>(av, p) = a;
    }
    if (KIND == K_AXPBY2) prescale<T>(av, (npass + C::VEC - 1) / C::VEC, s);
}

template <typename T, int KIND>
__device__ __forceinline__ void stage_drain_e(const Geom<T> &g, const Sc &s, unsigned char *buf,
                                              Chunk<T> (&av)[Cfg<T>::NPASS], int lane) {
    using C = Cfg<T>;
    constexpr int NE = C::NPASS * C::VEC;
    const LaneMap m = lane_map(g.nx, lane);
    if (m.c >= g.nx) return;
    const int npass = (g.ny + m.rpp - 1) / m.rpp;
#pragma unroll
    for (int p = 0; p < NE; ++p) {
        if (p >= npass) break;
        const int y = p * m.rpp + m.r0;
        if (y < g.ny) {
            const T b = g.transpose ? *slot_e<T>(buf, m.c, y) : *slot_e<T>(buf, y, m.c);
            g.dst[static_cast<int64_t>(y) * g.dld + m.c] = combine<KIND>(b, elem<T>(av, p), s);
        }
    }
}

// stage_drain_e for the kinds that do not read A.
template <typename T, int KIND>
__device__ __forceinline__ void stage_drain_e1(const Geom<T> &g, const Sc &s, unsigned char *buf, int lane) {
    static_assert(!kind_reads_a(KIND), "kinds that read A hold A in registers");
    const LaneMap m = lane_map(g.nx, lane);
    if (m.c >= g.nx) return;
#pragma unroll 4
    for (int y = m.r0; y < g.ny; y += m.rpp) {
        const T b = g.transpose ? *slot_e<T>(buf, m.c, y) : *slot_e<T>(buf, y, m.c);
        g.dst[static_cast<int64_t>(y) * g.dld + m.c] = combine<KIND>(b, T(), s);
    }
}

// Scalars of a problem in the kernel's form.
__device__ __forceinline__ void make_sc(const Scalars &S, Sc &s) {
    s.ar = S.alpha[0]; s.ai = S.alpha[1]; s.br = S.beta[0]; s.bi = S.beta[1];
    s.alpha_mid = mid_range(S.alpha[0]) && mid_range(S.alpha[1]);
    s.scal_mid = s.alpha_mid && mid_range(S.beta[0]) && mid_range(S.beta[1]);
    s.conj_mask = 0u;
    s.bexp = S.beta_exp;
    s.bsign_hi = static_cast<unsigned>(__double2hiint(S.beta[0])) & 0x80000000u;
    s.p2_add = static_cast<unsigned>(S.beta_exp) << 20;
    // admissible biased exponents e: e in [1, 2046] and e + k in [1, 2046]
    const int lo = max(1, 1 - S.beta_exp), hi = min(2046, 2046 - S.beta_exp);
    s.p2_lo = hi >= lo ? static_cast<unsigned>(lo) : 4096u;  // 4096: nothing admissible
    s.p2_span = hi >= lo ? static_cast<unsigned>(hi - lo) : 0u;
}

// The tile descriptors of one warp come in batches of 32: lane k holds the
// descriptor of the warp's tile 32 * b + k, loaded one batch ahead, and tile
// j is shuffled out of lane j % 32 of the current batch.
struct DescRegs {
    uint4 lo, hi;
};

template <bool MIS>
__device__ __forceinline__ DescRegs load_batch(const RemapLaunch &a, int64_t first, int64_t stride,
                                               int64_t b, int lane) {
    DescRegs r;
    const int64_t t = first + (b * 32 + lane) * stride;
    if (t < (MIS ? a.nmtiles : a.ntiles)) {
        const uint4 *p = reinterpret_cast<const uint4 *>((MIS ? a.mtiles : a.tiles) + t);
        r.lo = __ldg(p);
        r.hi = __ldg(p + 1);
    } else {
        r.lo = make_uint4(0, 0, 0, 0);
        r.hi = make_uint4(0, 0, 0, 0);
    }
    return r;
}

__device__ __forceinline__ TileDesc unpack_desc(const uint4 &lo, const uint4 &hi) {
    TileDesc d;
    d.src = (static_cast<uint64_t>(lo.y) << 32) | lo.x;
    d.dst = (static_cast<uint64_t>(lo.w) << 32) | lo.z;
    d.sld = static_cast<int32_t>(hi.x);
    d.dld = static_cast<int32_t>(hi.y);
    d.nx = static_cast<uint16_t>(hi.z & 0xFFFFu);
    d.ny = static_cast<uint16_t>(hi.z >> 16);
    d.prob = static_cast<uint16_t>(hi.w & 0xFFFFu);
    d.flags = static_cast<uint16_t>(hi.w >> 16);
    return d;
}

__device__ __forceinline__ TileDesc shfl_desc(const DescRegs &r, int src) {
    uint4 lo, hi;
    lo.x = __shfl_sync(0xffffffffu, r.lo.x, src);
    lo.y = __shfl_sync(0xffffffffu, r.lo.y, src);
    lo.z = __shfl_sync(0xffffffffu, r.lo.z, src);
    lo.w = __shfl_sync(0xffffffffu, r.lo.w, src);
    hi.x = __shfl_sync(0xffffffffu, r.hi.x, src);
    hi.y = __shfl_sync(0xffffffffu, r.hi.y, src);
    hi.z = __shfl_sync(0xffffffffu, r.hi.z, src);
    hi.w = __shfl_sync(0xffffffffu, r.hi.w, src);
    return unpack_desc(lo, hi);
}

template <typename T> __device__ __forceinline__ Geom<T> geom_of(const TileDesc &d) {
    Geom<T> g;
    g.src = reinterpret_cast<const T *>(d.src);
    g.dst = reinterpret_cast<T *>(d.dst);
    g.sld = d.sld;
    g.dld = d.dld;
    g.nx = d.nx;
    g.ny = d.ny;
    g.prob = d.prob;
    g.transpose = (d.flags & TF_TRANSPOSE) != 0;
    g.fast = (d.flags & TF_FAST) != 0;
    g.conj = ET<T>::CPLX && (d.flags & TF_CONJ) != 0;
    g.elem = (d.flags & TF_ELEM) != 0;
    return g;
}

// Walks the warp's tile sequence j = 0, 1, ... (tile first + j * stride).
struct TileStream {
    DescRegs cur, nxt;
    int64_t j;
};

// Next tile of the warp; false when none is left.  With per-problem scalars,
// tiles of problems of another kind are skipped (another launch covers
// them).  Called by all 32 lanes with the same state.
template <typename T, int KIND, bool MIS>
__device__ __forceinline__ bool next_tile(const RemapLaunch &a, int64_t first, int64_t stride,
                                          TileStream &ts, Geom<T> &g, int lane) {
    for (;;) {
        const int64_t t = first + ts.j * stride;
        if (t >= (MIS ? a.nmtiles : a.ntiles)) return false;
        const int k = static_cast<int>(ts.j & 31);
        if (k == 0 && ts.j > 0) {
            ts.cur = ts.nxt;
            ts.nxt = load_batch<MIS>(a, first, stride, (ts.j >> 5) + 1, lane);
        }
        const TileDesc d = shfl_desc(ts.cur, k);
        ++ts.j;
        if (a.per_problem && kind_of(a.per_problem[d.prob].flags) != KIND) continue;
        g = geom_of<T>(d);
        return true;
    }
}

// ---- the small-tile kernel ----
//
// Lists made mostly of small tiles (see split_small on the host) come as
// one-pass pieces (at most 32 chunks; piece_x x piece_y) in groups of at
// most group_pieces (a full tile's passes) of one problem.  A warp moves one
// group like one tile: it stages every piece's source into its own 512-byte
// slot, loads every piece's A chunk into its own register, waits once and
// drains every piece.  A warp thus keeps a full tile's bytes in flight
// instead of one small tile's.

// Row width (chunks) of a staged piece: the lanes per run of its lane map.
__device__ __forceinline__ int piece_width(int chunks) {
    return 1 << (chunks <= 1 ? 0 : 32 - __clz(chunks - 1));
}

// Stages a piece's source into its slot (one pass: every run has its lanes).
template <typename T>
__device__ __forceinline__ void piece_issue(const Geom<T> &g, unsigned char *slot_base, int lane) {
    using C = Cfg<T>;
    const int runs = g.transpose ? g.nx : g.ny;
    const int chunks = (g.transpose ? g.ny : g.nx) / C::VEC;
    const LaneMap m = lane_map(chunks, lane);
    const int W = piece_width(chunks);
    if (m.c < chunks && m.r0 < runs)
        cp_async16(slot_base + (m.r0 * W + (m.c ^ (swz<T>(m.r0) & (W - 1)))) * 16,
                   g.src + static_cast<int64_t>(m.r0) * g.sld + m.c * C::VEC);
}

// This lane's A chunk of a piece (zero when the lane has none).
template <typename T>
__device__ __forceinline__ Chunk<T> piece_load_a(const Geom<T> &g, int lane) {
    using C = Cfg<T>;
    const int chunks = g.nx / C::VEC;
    const LaneMap m = lane_map(chunks, lane);
    Chunk<T> a;
    a.raw = make_uint4(0, 0, 0, 0);
    if (m.c < chunks && m.r0 < g.ny) a = load_rw(g.dst + static_cast<int64_t>(m.r0) * g.dld + m.c * C::VEC);
    return a;
}

// Writes this lane's chunk of a staged piece to A.
template <typename T, int KIND>
__device__ __forceinline__ void piece_drain(const Geom<T> &g, const Sc &s, unsigned char *slot_base,
                                            const Chunk<T> &a, int lane) {
    using C = Cfg<T>;
    const int chunks = g.nx / C::VEC;
    const LaneMap m = lane_map(chunks, lane);
    const int y = m.r0;
    if (m.c >= chunks || y >= g.ny) return;
    const int x0 = m.c * C::VEC;
    Chunk<T> b;
    if (g.transpose) {
        // element (x0 + e, y): staged row x0 + e, chunk y / VEC, lane y % VEC
        const int W = piece_width(g.ny / C::VEC);
        if ((x0 + C::VEC - 1) * W >= 32) return;  // rows beyond one pass (never emitted by the host)
        const int cy = y / C::VEC, ey = y % C::VEC;
#pragma unroll
        for (int e = 0; e < C::VEC; ++e) {
            const int r = x0 + e;
            b.e[e] = reinterpret_cast<const T *>(slot_base + (r * W + (cy ^ (swz<T>(r) & (W - 1)))) * 16)[ey];
        }
    } else {
        const int W = piece_width(chunks);
        b.raw = *reinterpret_cast<const uint4 *>(slot_base + (y * W + (m.c ^ (swz<T>(y) & (W - 1)))) * 16);
    }
    Chunk<T> o;
#pragma unroll
    for (int e = 0; e < C::VEC; ++e) o.e[e] = combine<KIND>(b.e[e], a.e[e], s);
    store(g.dst + static_cast<int64_t>(y) * g.dld + x0, o);
}

#ifndef COSTA_SWARPS
#define COSTA_SWARPS 4
#endif
#ifndef COSTA_SMINB_4
#define COSTA_SMINB_4 5
#endif
#ifndef COSTA_SMINB_8
#define COSTA_SMINB_8 5
#endif
#ifndef COSTA_SMINB_8H
#define COSTA_SMINB_8H 3
#endif
#ifndef COSTA_SMINB_16
#define COSTA_SMINB_16 3
#endif
#ifndef COSTA_SMINB_16A
#define COSTA_SMINB_16A 2
#endif

// Launch shape of the small-tile kernel: warps per block and resident blocks
// per SM; each warp has one buffer of NS 512-byte slots.
template <typename T, int KIND> struct SCfg {
    static constexpr int WARPS = COSTA_SWARPS;
    static constexpr int MINB = sizeof(T) == 4 ? COSTA_SMINB_4
                              : sizeof(T) == 16 ? (KCfg<T, KIND>::READS_A ? COSTA_SMINB_16A : COSTA_SMINB_16)
                              : KCfg<T, KIND>::HEAVY ? COSTA_SMINB_8H : COSTA_SMINB_8;
    // pieces per group: the host's cap for the groups this kind receives
    static constexpr int NS = KCfg<T, KIND>::READS_A ? group_pieces_a(static_cast<int>(sizeof(T)), ET<T>::CPLX != 0)
                                                    : group_pieces(static_cast<int>(sizeof(T)));
    static constexpr int BUF_BYTES = NS * 512 + NS * 32;  // slots, then the group's descriptors
};

template <typename T, int KIND>
__global__ void __launch_bounds__(SCfg<T, KIND>::WARPS * 32, SCfg<T, KIND>::MINB)
    remap_small_kernel(const RemapLaunch args) {
    using SC = SCfg<T, KIND>;
    constexpr int NS = SC::NS;
    constexpr bool READS_A = KCfg<T, KIND>::READS_A;
    extern __shared__ __align__(128) unsigned char smem_raw[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    unsigned char *buf = smem_raw + warp * SC::BUF_BYTES;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * SC::WARPS;
    const int64_t first = static_cast<int64_t>(blockIdx.x) * SC::WARPS + warp;
    Sc s;
    int cached = -1;
    if (!args.per_problem) make_sc(args.s, s);
    for (int64_t gi = first; gi < args.ngroups; gi += stride) {
        const uint32_t g0 = __ldg(args.groups + gi), g1 = __ldg(args.groups + gi + 1);
        // 1 .. NS pieces (the host's groups); the clamp keeps the slots inside
        // this warp's buffer regardless
        const int cnt = min(static_cast<int>(g1 - g0), NS);
        // lane k copies piece k's descriptor next to the slots; every lane
        // then reads each descriptor with one broadcast load per half
        uint4 *dsm = reinterpret_cast<uint4 *>(buf + NS * 512);
        if (lane < cnt) {
            const uint4 *p = reinterpret_cast<const uint4 *>(args.pieces + g0 + lane);
            dsm[2 * lane] = __ldg(p);
            dsm[2 * lane + 1] = __ldg(p + 1);
        }
        __syncwarp();
        auto desc = [&](int k) { return unpack_desc(dsm[2 * k], dsm[2 * k + 1]); };
        if (args.per_problem) {  // one problem per group
            const int prob = static_cast<int>(desc(0).prob);
            if (kind_of(args.per_problem[prob].flags) != KIND) continue;
            if (prob != cached) {
                make_sc(args.per_problem[prob], s);
                cached = prob;
            }
        }
        for (int k = 0; k < cnt; ++k) piece_issue<T>(geom_of<T>(desc(k)), buf + 512 * k, lane);
        cp_async_commit();
        Chunk<T> av[NS];
        if (READS_A) {
#pragma unroll
            for (int k = 0; k < NS; ++k) {
                if (k >= cnt) break;  // uniform across the warp
                av[k] = piece_load_a<T>(geom_of<T>(desc(k)), lane);
            }
            if (KIND == K_AXPBY2) prescale<T>(av, cnt, s);
        }
        cp_async_wait<0>();
        __syncwarp();
#pragma unroll
        for (int k = 0; k < NS; ++k) {
            if (k >= cnt) break;
            const Geom<T> g = geom_of<T>(desc(k));
            s.conj_mask = g.conj ? 0x80000000u : 0u;
            piece_drain<T, KIND>(g, s, buf + 512 * k, av[k], lane);
        }
        __syncwarp();  // the slots are free before the next group is staged
    }
}

// Stages a tile's source: 16-byte chunks; in the instance for misaligned
// tiles (MIS), the runs' 16-byte windows or, for kinds that read A, single
// elements.
template <typename T, int KIND, bool MIS>
__device__ __forceinline__ void stage_any(const Geom<T> &g, unsigned char *buf, int lane) {
    if constexpr (MIS && KCfg<T, KIND>::READS_A) stage_issue_e<T>(g, buf, lane);
    else if constexpr (MIS) {
        if (sizeof(T) == 4 && g.elem) stage_issue_e<T>(g, buf, lane);  // the host flags 4-byte tiles only
        else stage_issue_w<T>(g, buf, lane);
    }
    else if (g.fast) stage_issue<T>(g, buf, lane);  // the element-wise fallback stages nothing
}

// Writes one staged tile.  `cached` holds the problem whose scalars are in
// `s`.
template <typename T, int KIND, int NB, bool MIS>
__device__ __forceinline__ void write_tile(const RemapLaunch &a, const Geom<T> &g, Sc &s, int &cached,
                                           unsigned char *buf, int lane) {
    using C = Cfg<T>;
    if (a.per_problem && g.prob != cached) {
        make_sc(a.per_problem[g.prob], s);
        cached = g.prob;
    }
    s.conj_mask = g.conj ? 0x80000000u : 0u;
    if constexpr (MIS && KCfg<T, KIND>::READS_A) {
        Chunk<T> av[C::NPASS];
        load_a_e<T, KIND>(g, s, av, lane);
        cp_async_wait<NB - 1>();  // this tile's copies (later tiles' may still fly)
        __syncwarp();
        stage_drain_e<T, KIND>(g, s, buf, av, lane);
    } else if constexpr (MIS) {
        cp_async_wait<NB - 1>();
        __syncwarp();
        if (sizeof(T) == 4 && g.elem) stage_drain_e1<T, KIND>(g, s, buf, lane);
        else stage_drain_w<T, KIND>(g, s, buf, lane);
    } else if (g.fast) {
        Chunk<T> av[C::NPASS];
        if constexpr (!drain_loads_a<T, KIND>()) load_a<T, KIND>(g, s, av, lane);
        cp_async_wait<NB - 1>();
        __syncwarp();
        stage_drain<T, KIND>(g, s, buf, av, lane);
    } else {
        tile_general<T, KIND>(g, s, buf, lane);
    }
    __syncwarp();  // the buffer is free before it is staged into again
}

// The tile kernel.  MIS = false moves the aligned ("fast") tiles of
// args.tiles with 16-byte chunks; MIS = true moves the tiles of args.mtiles
// (see "misaligned tiles" above): the misaligned ones and, in a list that
// is mostly misaligned, the aligned ones too, which its paths also move.  The host puts every tile in
// the right list, so no 16-byte access is ever made at a misaligned
// address.
template <typename T, int KIND, bool MIS>
__global__ void __launch_bounds__(KCfg<T, KIND, MIS>::WARPS * 32, KCfg<T, KIND, MIS>::MINB)
    remap_kernel(const RemapLaunch args) {
    using C = Cfg<T>;
    constexpr int NB = KCfg<T, KIND, MIS>::NBUF;
    constexpr int BB = MIS ? WCfg<T>::BUF_BYTES : C::BUF_BYTES;
    extern __shared__ __align__(128) unsigned char smem_raw[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    unsigned char *bufs = smem_raw + warp * NB * BB;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * C::WARPS;
    const int64_t first = static_cast<int64_t>(blockIdx.x) * C::WARPS + warp;

    Sc s;
    int cached = -1;
    if (!args.per_problem) make_sc(args.s, s);
    TileStream ts;
    ts.j = 0;
    ts.cur = load_batch<MIS>(args, first, stride, 0, lane);
    ts.nxt = load_batch<MIS>(args, first, stride, 1, lane);

    // ring[0] is the tile being written, ring[k] the tile k ahead, staged in
    // buffer (cur + k) % NB
    if constexpr (NB == 1) {  // no look-ahead: copy, wait, write, one tile at a time
        Geom<T> g;
        while (next_tile<T, KIND, MIS>(args, first, stride, ts, g, lane)) {
            stage_any<T, KIND, MIS>(g, bufs, lane);
            cp_async_commit();
            write_tile<T, KIND, 1, MIS>(args, g, s, cached, bufs, lane);
        }
        return;
    }
    Geom<T> ring[NB > 1 ? NB : 2];
    bool have[NB > 1 ? NB : 2];
#pragma unroll
    for (int k = 0; k < NB - 1; ++k) {
        have[k] = (k == 0 || have[k - 1]) && next_tile<T, KIND, MIS>(args, first, stride, ts, ring[k], lane);
        if (have[k]) stage_any<T, KIND, MIS>(ring[k], bufs + k * BB, lane);
        cp_async_commit();
    }
    int cur = 0;
    constexpr int LA = NB > 1 ? NB - 1 : 1;  // index of the look-ahead slot
    while (have[0]) {
        have[LA] = have[LA - 1] && next_tile<T, KIND, MIS>(args, first, stride, ts, ring[LA], lane);
        int ahead = cur + NB - 1;
        if (ahead >= NB) ahead -= NB;
        if (have[LA]) stage_any<T, KIND, MIS>(ring[LA], bufs + ahead * BB, lane);
        cp_async_commit();
        write_tile<T, KIND, NB, MIS>(args, ring[0], s, cached, bufs + cur * BB, lane);
#pragma unroll
        for (int k = 0; k < LA; ++k) {
            ring[k] = ring[k + 1];
            have[k] = have[k + 1];
        }
        cur = cur + 1 == NB ? 0 : cur + 1;
    }
    cp_async_wait<0>();
}

// ---- the TMA instance of the tile kernel (tma.cpp decides which tiles it takes) ----
//
// The same pipeline as the tile kernel without look-ahead, with the source
// staged by the TMA unit instead of per-lane cp.async copies: one lane
// issues the tile's boxes (cp.async.bulk.tensor, tensor maps passed by
// value in the launch) on the warp's mbarrier with the expected byte count,
// the warp loads its A chunks meanwhile, waits on the barrier's phase and
// drains the tile from the TMA layout.  The wait gives up after a bounded
// number of tries: it then counts the failure in args.err, waits once more
// for its copies, and ends the warp's work (no tile is written from a
// partial stage).

__device__ __forceinline__ unsigned smem_u32(const void *p) {
    return static_cast<unsigned>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(unsigned bar) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;\n" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void mbar_fence_init() { asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory"); }
__device__ __forceinline__ void mbar_expect_tx(unsigned bar, unsigned bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(unsigned bar, unsigned parity) {
    unsigned ok;
    asm volatile(
        "{\n"
        ".reg .pred p;\n"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
        "selp.u32 %0, 1, 0, p;\n"
        "}\n"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
// true once the barrier's phase `parity` has completed; false after the limit
__device__ __forceinline__ bool mbar_wait(unsigned bar, unsigned parity) {
    for (int i = 0; i < (1 << 22); ++i)
        if (mbar_try_wait(bar, parity)) return true;
    return false;
}
__device__ __forceinline__ void tma_load_2d(unsigned dst, const TmaMap *map, int x, int y, unsigned bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];\n" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
        : "memory");
}

// Lane 0: the tile's boxes on the warp's barrier (kept out of line, so that
// the registers of the A chunks held across the wait are not shared with
// this loop's).
template <typename T>
__device__ __noinline__ void tma_issue(const Geom<T> &g, const TmaMap *map, unsigned buf, unsigned bar) {
    const uint64_t c = reinterpret_cast<uint64_t>(g.src);
    const int x = static_cast<int>(c & 0xffffffffu), y = static_cast<int>(c >> 32);
    const int runs = g.transpose ? g.nx : g.ny;
    const int nbl = (g.transpose ? g.ny : g.nx) * static_cast<int>(sizeof(T)) / 128;
    mbar_expect_tx(bar, static_cast<unsigned>(runs * nbl * 128));
    for (int br = 0; br < runs / 16; ++br)
        for (int bl = 0; bl < nbl; ++bl)
            tma_load_2d(buf + (br * TCfg<T>::TBL + bl) * 2048, map, x + bl * 128, y + br * 16, bar);
}

struct TmaLaunch {
    RemapLaunch a;  // a.tiles / a.ntiles: the TMA tiles
    TmaMap maps[kMaxTmaMaps];
    unsigned int *err;
    int32_t nmaps;
};

#ifndef COSTA_TMA_MINB_8
#define COSTA_TMA_MINB_8 4
#endif
template <typename T, int KIND> struct TmaKCfg {
    static constexpr int MINB = sizeof(T) == 16 ? 3
                              : (sizeof(T) == 8 && COSTA_TMA_MINB_8 > 0) ? COSTA_TMA_MINB_8 : KCfg<T, KIND>::MINB;
};

template <typename T, int KIND>
__global__ void __launch_bounds__(Cfg<T>::WARPS * 32, TmaKCfg<T, KIND>::MINB)
    remap_tma_kernel(const __grid_constant__ TmaLaunch p) {
    using C = Cfg<T>;
    const RemapLaunch &args = p.a;
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    unsigned char *aligned = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    unsigned char *buf = aligned + warp * TCfg<T>::BUF;
    const unsigned bar = smem_u32(aligned + C::WARPS * TCfg<T>::BUF + warp * 8);
    if (lane == 0) {
        mbar_init(bar);
        mbar_fence_init();
    }
    __syncwarp();
    unsigned parity = 0;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * C::WARPS;
    const int64_t first = static_cast<int64_t>(blockIdx.x) * C::WARPS + warp;
    Sc s;
    int cached = -1;
    if (!args.per_problem) make_sc(args.s, s);
    TileStream ts;
    ts.j = 0;
    ts.cur = load_batch<false>(args, first, stride, 0, lane);
    ts.nxt = load_batch<false>(args, first, stride, 1, lane);
    Geom<T> g;
    while (next_tile<T, KIND, false>(args, first, stride, ts, g, lane)) {
        // g.src = (y << 32) | x: the source's (0, 0) in bytes along the run
        // (x) and runs (y) of tensor map g.sld
        if (g.sld < 0 || g.sld >= p.nmaps) {  // never listed by the host
            if (lane == 0) atomicAdd(p.err, 1u);
            continue;
        }
        if (lane == 0) tma_issue<T>(g, &p.maps[g.sld], smem_u32(buf), bar);
        if (args.per_problem && g.prob != cached) {
            make_sc(args.per_problem[g.prob], s);
            cached = g.prob;
        }
        s.conj_mask = g.conj ? 0x80000000u : 0u;
        Chunk<T> av[C::NPASS];
        if constexpr (!drain_loads_a<T, KIND>()) load_a<T, KIND>(g, s, av, lane);
        if (!mbar_wait(bar, parity)) {
            if (lane == 0) atomicAdd(p.err, 1u);
            mbar_wait(bar, parity);
            return;
        }
        parity ^= 1u;
        stage_drain<T, KIND, true>(g, s, buf, av, lane);
        __syncwarp();  // the buffer is free before the next tile's boxes land in it
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

template <typename T, int KIND, bool MIS>
cudaError_t launch_tiles(const RemapLaunch &a, cudaStream_t st) {
    auto kern = remap_kernel<T, KIND, MIS>;
    constexpr int kWarps = Cfg<T>::WARPS;
    const size_t smem = static_cast<size_t>(kWarps) * KCfg<T, KIND, MIS>::NBUF *
                        (MIS ? WCfg<T>::BUF_BYTES : Cfg<T>::BUF_BYTES);
    static int per_sm = 0;
    if (per_sm == 0) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(smem));
        if (e != cudaSuccess) return e;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kWarps * 32, smem);
        if (e != cudaSuccess) return e;
        if (per_sm < 1) per_sm = 1;
    }
    const int64_t n = MIS ? a.nmtiles : a.ntiles;
    const int64_t want = (n + kWarps - 1) / kWarps;
    const int64_t cap = static_cast<int64_t>(sm_count()) * per_sm;
    const int blocks = static_cast<int>(want < cap ? want : cap);
    if (blocks <= 0) return cudaSuccess;
    kern<<<blocks, kWarps * 32, smem, st>>>(a);
    count_launch();
    return cudaGetLastError();
}

template <typename T, int KIND>
cudaError_t launch_small(const RemapLaunch &a, cudaStream_t st) {
    using SC = SCfg<T, KIND>;
    auto kern = remap_small_kernel<T, KIND>;
    const size_t smem = static_cast<size_t>(SC::WARPS) * SC::BUF_BYTES;
    static int per_sm = 0;
    if (per_sm == 0) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(smem));
        if (e != cudaSuccess) return e;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, SC::WARPS * 32, smem);
        if (e != cudaSuccess) return e;
        if (per_sm < 1) per_sm = 1;
    }
    const int64_t want = (a.ngroups + SC::WARPS - 1) / SC::WARPS;
    const int64_t cap = static_cast<int64_t>(sm_count()) * per_sm;
    const int blocks = static_cast<int>(want < cap ? want : cap);
    if (blocks <= 0) return cudaSuccess;
    kern<<<blocks, SC::WARPS * 32, smem, st>>>(a);
    count_launch();
    return cudaGetLastError();
}

template <typename T, int KIND>
cudaError_t launch_tma(const RemapLaunch &a, cudaStream_t st) {
    const TmaLists &t = *a.tma;
    if (!t.maps || t.nmaps < 1 || t.nmaps > kMaxTmaMaps || !t.err) return cudaErrorInvalidValue;
    TmaLaunch p;
    p.a = a;
    p.a.tiles = t.ttiles;
    p.a.ntiles = t.nttiles;
    p.a.mtiles = nullptr;
    p.a.nmtiles = 0;
    p.a.ngroups = 0;
    p.a.tma = nullptr;
    for (int k = 0; k < kMaxTmaMaps; ++k) p.maps[k] = t.maps[k < t.nmaps ? k : 0];
    p.err = t.err;
    p.nmaps = t.nmaps;
    auto kern = remap_tma_kernel<T, KIND>;
    constexpr int kWarps = Cfg<T>::WARPS;
    const size_t smem = 1024 + static_cast<size_t>(kWarps) * (TCfg<T>::BUF + 8);
    static int per_sm = 0;
    if (per_sm == 0) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(smem));
        if (e != cudaSuccess) return e;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kWarps * 32, smem);
        if (e != cudaSuccess) return e;
        if (per_sm < 1) per_sm = 1;
    }
    const int64_t want = (t.nttiles + kWarps - 1) / kWarps;
    const int64_t cap = static_cast<int64_t>(sm_count()) * per_sm;
    const int blocks = static_cast<int>(want < cap ? want : cap);
    if (blocks <= 0) return cudaSuccess;
    kern<<<blocks, kWarps * 32, smem, st>>>(p);
    count_launch();
    return cudaGetLastError();
}

// The tile kernel over the aligned full-size tiles, then over the
// misaligned ones, then the small-tile kernel over the groups of pieces
// (each launched only when it has work).
template <typename T, int KIND>
cudaError_t launch_t(const RemapLaunch &a, cudaStream_t st) {
    // 16-byte elements sit at 16-byte aligned addresses, so every tile of
    // theirs is aligned and their misaligned instance is not built
    if (sizeof(T) == 16 && a.nmtiles > 0) return cudaErrorInvalidValue;
    cudaError_t e = a.ntiles > 0 ? launch_tiles<T, KIND, false>(a, st) : cudaSuccess;
    if (e == cudaSuccess && a.tma && a.tma->nttiles > 0) e = launch_tma<T, KIND>(a, st);
    if constexpr (sizeof(T) != 16)
        if (e == cudaSuccess && a.nmtiles > 0) e = launch_tiles<T, KIND, true>(a, st);
    if (e == cudaSuccess && a.ngroups > 0) e = launch_small<T, KIND>(a, st);
    return e;
}

// Kernel for (element type, combine kind).  Real types never take K_CPLX or
// K_CSCALE.
template <typename T>
cudaError_t launch_remap_t(const RemapLaunch &a, int kind, cudaStream_t st) {
    switch (kind) {
    case K_COPY: return launch_t<T, K_COPY>(a, st);
    case K_SCALE: return launch_t<T, K_SCALE>(a, st);
    case K_AXPBY: return launch_t<T, K_AXPBY>(a, st);
    case K_AXPBY2: return launch_t<T, K_AXPBY2>(a, st);
    case K_CPLX:
        if constexpr (ET<T>::CPLX) return launch_t<T, K_CPLX>(a, st);
        return cudaErrorInvalidValue;
    case K_CSCALE:
        if constexpr (ET<T>::CPLX) return launch_t<T, K_CSCALE>(a, st);
        return cudaErrorInvalidValue;
    default:
        return cudaErrorInvalidValue;
    }
}

}  // namespace remap
}  // namespace costa
