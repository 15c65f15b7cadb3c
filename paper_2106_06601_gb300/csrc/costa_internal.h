// Internal types shared by the host planner (costa.cpp) and the kernels
// (remap_*.cu, volume.cu and the other .cu files).  Not part of the public ABI.
#pragma once

#include <cstdint>
#include <vector>

#include <cuda_runtime_api.h>

#ifdef __CUDACC__
#define COSTA_HD __host__ __device__
#else
#define COSTA_HD
#endif

#include "costa_gb300.h"

namespace costa {

// Storage of one block as the kernels see it (Sec. 6, Fig. 1).
struct DevBlock {
    uint64_t ptr;   // device address of element (0, 0)
    int32_t ld;     // leading dimension (elements)
    int32_t order;  // 0 column-major, 1 row-major
};
static_assert(sizeof(DevBlock) == 16, "DevBlock layout");

}  // namespace costa

// A layout as the library holds it (host copies of the description).
struct costa_layout_s {
    uint64_t id;
    costa_dtype dt;
    int nranks;
    int nbr, nbc;
    int64_t m, n;
    std::vector<int64_t> R, C;
    std::vector<int32_t> owner;
    std::vector<costa::DevBlock> blocks;
    int checked_device = -1;  // device whose access to every block was checked
};

namespace costa {

// One piece of a grid-overlay interval along one axis (rows or columns of A),
// at most the kernel tile extent long.  The overlay (Sec. 5, "Grid Overlay")
// is the product of the row intervals and the column intervals, so the
// kernel's tile grid is the product of the row pieces and the column pieces.
struct AxisTile {
    int32_t a_blk;  // block index of A along this axis
    int32_t b_blk;  // block index of op(B) along this axis (a B row block for
                    // A's rows when op = N, a B column block when op = T/C)
    int32_t a_off;  // offset of the piece inside A's block
    int32_t b_off;  // offset of the piece inside op(B)'s block
    int32_t len;    // extent of the piece
    int32_t cell;   // index of the overlay interval it belongs to
};
static_assert(sizeof(AxisTile) == 24, "AxisTile layout");

// One grid-overlay interval along one axis (used by the volume kernel).
struct Interval {
    int32_t a_blk;
    int32_t b_blk;
    int64_t len;
};

// One tile of the remap kernel, resolved on the host at plan time: a
// rectangle inside one block of A and one block of B (or a staging region),
// in its canonical frame x = the target's contiguous axis:
//   target element (x, y) at dst + (x + y * dld) elements
//   source element (x, y) at src + (x + y * sld) elements (copy tile)
//                         or src + (x * sld + y) elements (transposed tile)
struct TileDesc {
    // Left uninitialized: tile lists are sized first and then filled in
    // place, in parallel, so zeroing them would only add a serial pass.
    COSTA_HD TileDesc() {}
    uint64_t src;    // device address of source element (0, 0)
    uint64_t dst;    // device address of target element (0, 0)
    int32_t sld;     // source stride (elements)
    int32_t dld;     // target stride (elements)
    uint16_t nx, ny; // extents, at most the tile extent
    uint16_t prob;   // problem index within the launch
    uint16_t flags;  // TF_*
};
static_assert(sizeof(TileDesc) == 32, "TileDesc layout");
enum : uint16_t { TF_TRANSPOSE = 1, TF_FAST = 2, TF_CONJ = 4, TF_ELEM = 8 };

// Scalars of one problem, as doubles ({re, im}); float data carries values
// that are exactly representable in float.
struct Scalars {
    double alpha[2];
    double beta[2];
    int32_t flags;
    int32_t beta_exp;  // k with |beta| = 2^k when SF_BPOW2 is set
};
enum : int32_t { SF_BETA0 = 1, SF_ALPHA1 = 2, SF_CPLX = 4, SF_BPOW2 = 8 };

// Combine kinds: each kernel is compiled for one, so every path keeps only
// the registers it needs.
//   K_COPY  alpha = 1, beta = 0        out = op(b)
//   K_SCALE real alpha, beta = 0       out = alpha * op(b)
//   K_AXPBY real alpha, beta != 0      out = fma(alpha, op(b), beta * a)
//   K_CPLX  complex beta (or complex alpha with beta != 0): each component
//           a compensated sum of its four products (Dot2)
//   K_AXPBY2 as K_AXPBY with beta = +-2^k: beta * a is formed exactly on the
//            integer pipes (exponent add), saving one multiply on the scarce
//            FP64 pipe; same bits as K_AXPBY
//   K_CSCALE complex alpha, beta = 0   out = alpha * op(b) by Dot2 (double
//            data in the middle range: Kahan's 2 x 2 determinant algorithm);
//            A is not read (BLAS convention), so NaN in A does not propagate
enum : int { K_COPY = 0, K_SCALE = 1, K_AXPBY = 2, K_CPLX = 3, K_AXPBY2 = 4, K_CSCALE = 5, K_NKINDS = 6 };

// The kinds whose output depends on A's old value (beta != 0).
COSTA_HD constexpr bool kind_reads_a(int kind) { return kind == K_AXPBY || kind == K_CPLX || kind == K_AXPBY2; }

COSTA_HD inline int kind_of(int32_t flags) {
    if (flags & SF_CPLX) return (flags & SF_BETA0) ? K_CSCALE : K_CPLX;
    if (!(flags & SF_BETA0)) return (flags & SF_BPOW2) ? K_AXPBY2 : K_AXPBY;
    if (!(flags & SF_ALPHA1)) return K_SCALE;
    return K_COPY;
}


// A tensor map (CUtensorMap: 128 opaque bytes, 64-byte aligned) for the
// TMA-staged tiles; at most kMaxTmaMaps per launch, passed by value.
struct alignas(64) TmaMap {
    unsigned long long opaque[16];
};
constexpr int kMaxTmaMaps = 4;

// Aligned full-size tiles whose source is staged by TMA (the TMA instance of
// the tile kernel): each TileDesc's src holds (y << 32) | x, the byte
// coordinates of the source's (0, 0) in tensor map sld of `maps`.
struct TmaLists {
    const TileDesc *ttiles;
    int64_t nttiles;
    const TmaMap *maps;   // host array of nmaps maps (copied into the launch)
    int32_t nmaps;
    unsigned int *err;    // device word: TMA waits that gave up (0 when none)
};

struct RemapLaunch {
    const TileDesc *tiles;       // aligned full-size tiles (the tile kernel)
    int64_t ntiles;
    const TileDesc *mtiles;      // misaligned tiles (the tile kernel's second instance)
    int64_t nmtiles;
    const TileDesc *pieces;      // one-pass pieces of small tiles (the small-tile kernel)
    const uint32_t *groups;      // group g = pieces [groups[g], groups[g + 1])
    int64_t ngroups;
    int32_t dtype;
    int32_t pad;
    const Scalars *per_problem;  // device array indexed by TileDesc::prob, or nullptr: use `s`
    Scalars s;
    // host only: the TMA-staged tiles of this launch, or null.  A pointer
    // keeps this struct (the kernels' parameter) at 120 bytes; 40 bytes more
    // of parameters made ptxas spill more in the tile kernel.
    const struct TmaLists *tma;
};

struct VolumeProblemDev {
    const Interval *rows;
    const Interval *cols;
    const int32_t *ownerA;      // nbrA * nbcA
    const int32_t *ownerB;      // nbrB * nbcB
    int64_t cell_begin;
    int32_t nr, nc;
    int32_t nbcA, nbcB;
    int32_t op;
    int32_t pad;
};

struct VolumeLaunch {
    const VolumeProblemDev *probs;
    int32_t nprob;
    int32_t P;
    int64_t total_cells;
    unsigned long long *V;      // P * P, zeroed by the caller
};

// Tile extent (elements along each axis of A) for an element size; shared
// by the planner and the kernels.
#ifndef COSTA_TS_16
#define COSTA_TS_16 32
#endif
#ifndef COSTA_TS_4
#define COSTA_TS_4 32
#endif
COSTA_HD constexpr int tile_extent(int esize) { return esize == 16 ? COSTA_TS_16 : esize == 4 ? COSTA_TS_4 : 32; }
static_assert(tile_extent(4) <= 32 && tile_extent(16) <= 32, "the kernels' lane maps need tiles of at most 32");

// Small tiles are cut by the host into pieces of at most piece_x x piece_y
// elements, each exactly one warp pass (32 lanes x 16 bytes at most), and
// grouped at most group_pieces (a full tile's tile_passes) per group, one
// problem per group; the small-tile kernel moves a group like one tile.
COSTA_HD constexpr int piece_x(int esize) { return esize == 4 ? 16 : 8; }
COSTA_HD constexpr int piece_y(int esize) { return esize == 16 ? 4 : 8; }
COSTA_HD constexpr int tile_passes(int esize) { return tile_extent(esize) * tile_extent(esize) * esize / 512; }
#ifndef COSTA_GROUP_4
#define COSTA_GROUP_4 8
#endif
COSTA_HD constexpr int group_pieces(int esize) { return esize == 4 ? COSTA_GROUP_4 : tile_passes(esize); }
// Groups for the kinds that read A, of 8-byte types: smaller (measured on
// GB300, 8192^2 T, BC8: f64 86 -> 91% of copy at 8 pieces, c64 87 -> 93% at
// 12; the copy kind loses 10-15% on groups below 16, so it keeps those).
#ifndef COSTA_GROUP_8A
#define COSTA_GROUP_8A 8
#endif
#ifndef COSTA_GROUP_8CA
#define COSTA_GROUP_8CA 12
#endif
COSTA_HD constexpr int group_pieces_a(int esize, bool cplx) {
    return esize == 8 ? (cplx ? COSTA_GROUP_8CA : COSTA_GROUP_8A) : group_pieces(esize);
}
static_assert(group_pieces_a(8, false) <= group_pieces(8) && group_pieces_a(8, true) <= group_pieces(8),
              "a group must fit the small-tile kernel's slots");

// Launches the remap kernel for (args.dtype, kind) over a tile list.  With
// args.per_problem set, the kernel skips the tiles of problems of another kind.
cudaError_t launch_remap(const RemapLaunch &args, int kind, cudaStream_t stream);
cudaError_t launch_remap_f32(const RemapLaunch &args, int kind, cudaStream_t stream);
cudaError_t launch_remap_f64(const RemapLaunch &args, int kind, cudaStream_t stream);
cudaError_t launch_remap_c64(const RemapLaunch &args, int kind, cudaStream_t stream);
cudaError_t launch_remap_c128(const RemapLaunch &args, int kind, cudaStream_t stream);
cudaError_t launch_volume(const VolumeLaunch &args, cudaStream_t stream);
void count_launch();
int64_t launches_so_far();

// Error reporting and pair validation shared with entry points defined
// outside costa.cpp.
costa_status report_error(costa_status s, const char *message);
costa_status check_pair(const costa_layout_s *A, const costa_layout_s *B, int op);

}  // namespace costa
