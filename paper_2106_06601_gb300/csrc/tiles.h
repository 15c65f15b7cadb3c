// Tile planning shared by the plan builder and the diagnostics: the grid
// overlay per axis (Sec. 5, "Grid Overlay"), the tile list of the remap
// kernel and its order, and the split of small tiles into one-pass pieces for
// the small-tile kernel.  Host code only.
#pragma once

#include <algorithm>
#include <cstdint>
#include <thread>
#include <utility>
#include <vector>

#include "costa_internal.h"

namespace costa {

int super_tile(int esize);

// Element size in bytes of a costa_dtype (0 for an unknown type).
inline int esize_of(int dt) {
    switch (dt) {
    case COSTA_F32: return 4;
    case COSTA_F64: return 8;
    case COSTA_C64: return 8;
    case COSTA_C128: return 16;
    default: return 0;
    }
}

// ---------------------------------------------------------------------------
// Grid overlay along one axis (Sec. 5): the sorted union of A's splits and
// op(B)'s splits cuts the axis into intervals, each inside exactly one block
// of A and one block of op(B) (the unique cover).  Empty blocks are skipped.
// ---------------------------------------------------------------------------
struct AxisCut {
    std::vector<Interval> intervals;
    std::vector<AxisTile> tiles;
};

struct ProblemHost {
    const costa_layout_s *A;
    const costa_layout_s *B;
    costa_op op;
    AxisCut rows, cols;
};

// ---- host threads for plan building ----
//
// parallel_for(n, grain, f) calls f(begin, end) on up to plan_threads()
// contiguous chunks of [0, n), the calling thread taking the first.  It is
// used only where every chunk writes its own precomputed output range, so a
// plan does not depend on the number of threads.  COSTA_PLAN_THREADS sets the
// thread count (default: the hardware threads, at most 16).
int plan_threads();

inline thread_local bool t_in_parallel = false;  // nested parallel_for calls run serially

template <typename F> void parallel_for(int64_t n, int64_t grain, F &&f) {
    const int64_t chunks = std::min<int64_t>(plan_threads(), (n + grain - 1) / std::max<int64_t>(grain, 1));
    if (chunks <= 1 || t_in_parallel) {
        if (n > 0) f(int64_t(0), n);
        return;
    }
    std::vector<std::thread> workers;
    workers.reserve(static_cast<size_t>(chunks - 1));
    for (int64_t c = 1; c < chunks; ++c)
        workers.emplace_back([&f, n, c, chunks] {
            t_in_parallel = true;
            f(n * c / chunks, n * (c + 1) / chunks);
        });
    t_in_parallel = true;
    f(int64_t(0), n / chunks);
    t_in_parallel = false;
    for (std::thread &w : workers) w.join();
}

// A tile list split between the remap kernels: aligned and misaligned
// full-size tiles for the two instances of the tile kernel, and the one-pass
// pieces of the small tiles with their groups for the small-tile kernel.
struct SplitList {
    std::vector<TileDesc> big;  // aligned ("fast") full-size tiles
    std::vector<TileDesc> mis;  // misaligned tiles (16-byte windows or single elements)
    std::vector<TileDesc> pieces;
    std::vector<uint32_t> groups;  // group g = pieces [groups[g], groups[g + 1])
    std::vector<uint32_t> groups_a;  // the same pieces in the groups of the kinds that read A
    int64_t ngroups() const { return groups.empty() ? 0 : static_cast<int64_t>(groups.size()) - 1; }
    int64_t ngroups_a() const { return groups_a.empty() ? 0 : static_cast<int64_t>(groups_a.size()) - 1; }
};

// Visits the tiles of a problem in the global super-tile order (see
// super_tile in tiles.cpp), calling f(row piece, column piece).
template <typename F> void for_each_tile(const ProblemHost &ph, F &&f) {
    const int kSuper = super_tile(esize_of(ph.A->dt));
    const int nu = static_cast<int>(ph.rows.tiles.size()), nv = static_cast<int>(ph.cols.tiles.size());
    for (int su = 0; su < nu; su += kSuper)
        for (int sv = 0; sv < nv; sv += kSuper)
            for (int v = sv; v < std::min(sv + kSuper, nv); ++v)
                for (int u = su; u < std::min(su + kSuper, nu); ++u) f(ph.rows.tiles[u], ph.cols.tiles[v]);
}

AxisCut cut_axis(const std::vector<int64_t> &SA, const std::vector<int64_t> &SB, int64_t extent, int ts, int vec,
                 bool align_a);
AxisCut cut_pair_axis(const costa_layout_s *A, const costa_layout_s *B, int op, int axis, int ts);

bool aligned16(uint64_t addr, int64_t ld_bytes);
TileDesc direct_tile(const ProblemHost &ph, const AxisTile &rt, const AxisTile &ct, int es, int prob);
void set_fast(TileDesc &d, int es);

// True when misaligned tiles (with target_only, tiles whose target runs are
// misaligned) hold at least half of the elements.
bool mostly_misaligned(const TileDesc *tiles, size_t n, int es, bool target_only);
// Whether a problem's tiles take the target-local order; `tiles` are the
// problem's tiles (their alignment flags set).
bool use_local_order(const ProblemHost &ph, const TileDesc *tiles, size_t n);
void radix_sort_pairs(std::vector<std::pair<uint64_t, uint32_t>> &v);
void order_tiles_local(std::vector<TileDesc> &list, size_t first, size_t last, int es, int ts);
void append_direct_tiles(const ProblemHost &ph, int prob, int es, int ts, std::vector<TileDesc> &list);

int next_pow2(int v);
int fast_tile_passes(const TileDesc &d, int es);
int small_limit(int es);
bool is_small(const TileDesc &d, int es);
int cut_pieces(const TileDesc &d, int es, TileDesc *out);
SplitList split_small(std::vector<TileDesc> &&list, int es, bool cplx);

// The aligned tiles of problems k with halve[k] that are wider than hx
// along x (A's contiguous axis) and at least 2 hx high, cut into [0, hx)
// and the rest along x, in list order (the two halves of a tile adjacent);
// empty when no tile is cut.  hx * es must be a multiple of 16, so both
// halves stay 16-byte aligned.
std::vector<TileDesc> split_x_halves(const std::vector<TileDesc> &list, int hx, int es,
                                     const std::vector<char> &halve);

// Whether a problem's aligned tiles are also listed as x-halves: for 4- and
// 8-byte types, when A's blocks are at most 256 elements along A's
// contiguous axis, and, for 8-byte types, when op transposes.  Every f32
// kind runs on the halves, and the f64 / c64 axpby kind with beta = +-2^k.
bool use_halves(const ProblemHost &ph, int es);

}  // namespace costa
