// Tile planning: the grid overlay per axis, the remap kernel's tile list
// and its order, and the one-pass pieces of small tiles (declarations and
// the reasons behind each choice in tiles.h and below).
#include "tiles.h"

#include <atomic>
#include <cstdlib>
#include <cstring>

namespace costa {

// Cuts one axis into pieces of at most ts elements.  When an interval starts
// off a 16-byte boundary (vec elements) of the side chosen by `align_a`
// (A's block if true, else op(B)'s), one short first piece reaches the
// boundary, so that the remaining pieces start aligned and can use vector
// accesses; otherwise the pieces are ts long from the interval's start.
AxisCut cut_axis(const std::vector<int64_t> &SA, const std::vector<int64_t> &SB, int64_t extent,
                 int ts, int vec, bool align_a) {
    AxisCut out;
    const int nA = static_cast<int>(SA.size()) - 1, nB = static_cast<int>(SB.size()) - 1;
    int ka = 0, kb = 0;
    int64_t pos = 0;
    while (pos < extent) {
        while (ka + 1 < nA && SA[ka + 1] <= pos) ++ka;
        while (kb + 1 < nB && SB[kb + 1] <= pos) ++kb;
        const int64_t end = std::min(SA[ka + 1], SB[kb + 1]);
        const int64_t len = end - pos;
        const int cell = static_cast<int>(out.intervals.size());
        out.intervals.push_back(Interval{ka, kb, len});
        const int64_t a0 = pos - SA[ka], b0 = pos - SB[kb];
        int64_t q = 0;
        const int64_t phase = (align_a ? a0 : b0) % vec;
        while (q < len) {
            const int64_t want = (q == 0 && phase != 0) ? vec - phase : ts;
            const int64_t piece = std::min<int64_t>(want, len - q);
            out.tiles.push_back(AxisTile{ka, kb, static_cast<int32_t>(a0 + q),
                                         static_cast<int32_t>(b0 + q),
                                         static_cast<int32_t>(piece), cell});
            q += piece;
        }
        pos = end;
    }
    return out;
}

// Cuts axis 0 (rows) or 1 (columns) of A for the pair (A, op(B)).  Each axis
// is aligned to the side whose contiguous axis it is (decided by the first
// block's order: column-major makes rows contiguous), so that side's runs
// start on 16-byte boundaries.
AxisCut cut_pair_axis(const costa_layout_s *A, const costa_layout_s *B, int op, int axis, int ts) {
    const bool tr = op != COSTA_OP_N;
    const int vec = 16 / esize_of(A->dt);
    const bool a_rows_fast = A->blocks.empty() || A->blocks[0].order == COSTA_COL_MAJOR;
    const bool b_col = B->blocks.empty() || B->blocks[0].order == COSTA_COL_MAJOR;
    const bool b_rows_fast = tr ? !b_col : b_col;  // op(B)'s contiguous axis is rows
    if (axis == 0) return cut_axis(A->R, tr ? B->C : B->R, A->m, ts, vec, a_rows_fast || !b_rows_fast);
    return cut_axis(A->C, tr ? B->R : B->C, A->n, ts, vec, !a_rows_fast || b_rows_fast);
}

int plan_threads() {
    static const int t = [] {
        const char *e = std::getenv("COSTA_PLAN_THREADS");
        int v = e ? std::atoi(e) : 0;
        if (v < 1) v = static_cast<int>(std::min(16u, std::max(1u, std::thread::hardware_concurrency())));
        return std::min(v, 64);
    }();
    return t;
}

int next_pow2(int v) {
    int p = 1;
    while (p < v) p <<= 1;
    return p;
}

// Warp passes the tile kernel needs for a fast tile: the larger of its
// staging and drain pass counts, with the kernel's lane maps (a run of c
// chunks takes the next power of two >= c lanes; 32 lanes per pass).
int fast_tile_passes(const TileDesc &d, int es) {
    const int vec = 16 / es;
    const bool tr = (d.flags & TF_TRANSPOSE) != 0;
    const int runs = tr ? d.nx : d.ny;
    const int rpp_s = 32 / next_pow2((tr ? d.ny : d.nx) / vec);
    const int rpp_d = 32 / next_pow2(d.nx / vec);
    return std::max((runs + rpp_s - 1) / rpp_s, (d.ny + rpp_d - 1) / rpp_d);
}



// A small tile is a fast tile needing fewer passes than small_limit: half
// of a full tile's passes (so 16 x 16 tiles of every element type are small).
int small_limit(int es) { return tile_passes(es) / 2; }

// Share (percent) of a list's elements that small tiles must hold for the
// list to use the small-tile kernel.
#ifndef COSTA_SMALL_SHARE
#define COSTA_SMALL_SHARE 50
#endif

bool is_small(const TileDesc &d, int es) {
    // a pass moves at most 32 chunks: a larger tile cannot be small
    const int64_t area = static_cast<int64_t>(d.nx) * d.ny;
    if (area * es >= int64_t(512) * small_limit(es) || !(d.flags & TF_FAST)) return false;
    return fast_tile_passes(d, es) < small_limit(es);
}

// Splits a list between the kernels.  Only a list whose small tiles hold at
// least half of its elements uses the small-tile kernel: in a mixed list the
// warps on small tiles wait on latency while the others keep DRAM busy, and
// one launch over the whole list measured faster than two (c4: 6157 against
// 5787 GB/s).  A small tile is cut into pieces of at most piece_x x piece_y
// (x fastest, so that consecutive pieces continue the target's runs); piece
// offsets are multiples of the 16-byte chunk, so the pieces stay on the
// vector path.  Pieces are grouped in list order, at most group_pieces(es)
// per group and one problem per group.
// Cuts a small tile into its pieces (writing them to `out` when non-null);
// returns the number of pieces, or -1 if a piece would leave the vector path
// (not expected for a fast tile).
int cut_pieces(const TileDesc &d, int es, TileDesc *out) {
    const int px = piece_x(es), py = piece_y(es);
    const bool tr = (d.flags & TF_TRANSPOSE) != 0;
    int k = 0;
    for (int y0 = 0; y0 < d.ny; y0 += py)
        for (int x0 = 0; x0 < d.nx; x0 += px, ++k) {
            if (!out) continue;
            TileDesc pc = d;
            pc.nx = static_cast<uint16_t>(std::min(px, d.nx - x0));
            pc.ny = static_cast<uint16_t>(std::min(py, d.ny - y0));
            pc.dst = d.dst + static_cast<uint64_t>((x0 + static_cast<int64_t>(y0) * d.dld) * es);
            pc.src = d.src + static_cast<uint64_t>(
                                 (tr ? static_cast<int64_t>(x0) * d.sld + y0 : x0 + static_cast<int64_t>(y0) * d.sld) * es);
            set_fast(pc, es);
            if (!(pc.flags & TF_FAST)) return -1;
            out[k] = pc;
        }
    return k;
}

// Measured on GB300, same box, halves against whole 32 x 32 tiles:
//  - f32, 8192^2, BC64 -> BC128: T copy 81 -> 89%, T beta=0.5 88 -> 91%,
//    N copy 84 -> 91% of the copy bandwidth; c4 6243 -> 6372 GB/s, with its
//    32 x 16 tiles left whole (halving them too cost c4 7%);
//  - f64 T, BC64 -> BC128, beta=0.5 (c2): 6184 -> 6338 GB/s; c64 T +8%;
//  - lost: the other 8-byte kinds (f64 T copy 91 -> 87%), c128 (95 -> 86%),
//    op = N for 8-byte types (no gain), and targets of whole panels
//    (1024- and 4096-row blocks: 2-6%).
bool use_halves(const ProblemHost &ph, int es) {
    if (es != 4 && es != 8) return false;
    const costa_layout_s *a = ph.A;
    const bool rows_fast = a->blocks.empty() || a->blocks[0].order == COSTA_COL_MAJOR;
    const std::vector<int64_t> &S = rows_fast ? a->R : a->C;
    int64_t widest = 0;
    for (size_t i = 0; i + 1 < S.size(); ++i) widest = std::max(widest, S[i + 1] - S[i]);
    return widest <= 256 && (es == 4 || ph.op != COSTA_OP_N);
}

std::vector<TileDesc> split_x_halves(const std::vector<TileDesc> &list, int hx, int es,
                                     const std::vector<char> &halve) {
    const int64_t n = static_cast<int64_t>(list.size());
    auto cut = [&](const TileDesc &d) { return d.nx > hx && d.ny >= 2 * hx && halve[d.prob]; };
    std::vector<int64_t> pos(static_cast<size_t>(n) + 1, 0);
    for (int64_t i = 0; i < n; ++i) pos[i + 1] = pos[i] + (cut(list[i]) ? 2 : 1);
    std::vector<TileDesc> out;
    if (pos[n] == n) return out;
    out.resize(static_cast<size_t>(pos[n]));
    parallel_for(n, 1 << 15, [&](int64_t a, int64_t b) {
        for (int64_t i = a; i < b; ++i) {
            const TileDesc &d = list[i];
            TileDesc *o = &out[static_cast<size_t>(pos[i])];
            o[0] = d;
            if (!cut(d)) continue;
            const bool tr = (d.flags & TF_TRANSPOSE) != 0;
            o[0].nx = static_cast<uint16_t>(hx);
            o[1] = d;
            o[1].nx = static_cast<uint16_t>(d.nx - hx);
            o[1].dst = d.dst + static_cast<uint64_t>(hx) * es;
            o[1].src = d.src + static_cast<uint64_t>(tr ? static_cast<int64_t>(hx) * d.sld : hx) * es;
        }
    });
    return out;
}

bool mostly_misaligned(const TileDesc *tiles, size_t n, int es, bool target_only) {
    int64_t mis = 0, all = 0;
    for (size_t i = 0; i < n; ++i) {
        const TileDesc &d = tiles[i];
        const int64_t e = static_cast<int64_t>(d.nx) * d.ny;
        all += e;
        const bool m = target_only ? !aligned16(d.dst, static_cast<int64_t>(d.dld) * es) || d.nx % (16 / es) != 0
                                   : !(d.flags & TF_FAST);
        if (m) mis += e;
    }
    return n > 0 && 2 * mis >= all;
}

SplitList split_small(std::vector<TileDesc> &&all, int es, bool cplx) {
    SplitList out;
    // misaligned tiles go to their own instance of the tile kernel
    std::vector<TileDesc> list;
    {
        size_t nmis = 0;
        for (const TileDesc &d : all) nmis += (d.flags & TF_FAST) ? 0 : 1;
        if (nmis == 0) {
            list = std::move(all);
        } else {
            // When most of the list is misaligned (odd block sizes), its
            // aligned tiles go to the misaligned instance too: an aligned
            // tile and its misaligned neighbour along the target's runs
            // share the 32-byte sectors where they meet, and in two
            // launches the first half of such a sector is evicted before
            // the second arrives (a DRAM read-modify-write).  Measured on
            // GB300, 8192^2 T, BC50 -> BC75 (88% of the elements
            // misaligned), GB/s two launches -> one: f64 copy 4255 -> 4606,
            // scale 4249 -> 4689, c64 copy 4251 -> 4596.
            const bool one_list = mostly_misaligned(all.data(), all.size(), es, false);
            if (one_list) {
                out.mis = std::move(all);
            } else {
                list.reserve(all.size() - nmis);
                out.mis.reserve(nmis);
                for (const TileDesc &d : all) ((d.flags & TF_FAST) ? list : out.mis).push_back(d);
            }
            // 4-byte tiles whose target runs are misaligned take the
            // one-element-per-lane path in every kind (TF_ELEM): one warp
            // store then writes a whole target run, the partial 32-byte
            // sectors at its ends included, where the window path writes
            // the partial chunks in a second pass.  Measured on GB300,
            // 8192^2 T copy, BC64 -> BC128, GB/s window -> element: A's ld
            // = 1 mod 4 3586 -> 4320 (N: 3695 -> 4378), both lds odd 3675 ->
            // 4380, BC50 -> BC75 2235 -> 2455; B's ld odd alone 5300 ->
            // 4760 (so the window path keeps it); 8-byte types lose 5-15%.
            if (es == 4) {
                for (TileDesc &d : out.mis)
                    if (!aligned16(d.dst, static_cast<int64_t>(d.dld) * es) || d.nx % 4 != 0)
                        d.flags = static_cast<uint16_t>(d.flags | TF_ELEM);
            }
        }
    }
    const int64_t n = static_cast<int64_t>(list.size());
    std::vector<int32_t> npc(static_cast<size_t>(n));  // pieces of a small tile, 0 for the others
    parallel_for(n, 1 << 15, [&](int64_t a, int64_t b) {
        for (int64_t i = a; i < b; ++i) npc[i] = is_small(list[i], es) ? cut_pieces(list[i], es, nullptr) : 0;
    });
    int64_t small_elems = 0, all_elems = 0;
    for (int64_t i = 0; i < n; ++i) {
        const int64_t e = static_cast<int64_t>(list[i].nx) * list[i].ny;
        all_elems += e;
        if (npc[i] > 0) small_elems += e;
    }
    if (100 * small_elems < COSTA_SMALL_SHARE * all_elems || small_elems == 0) {
        out.big = std::move(list);
        return out;
    }
    // positions: pieces of small tile i at poff[i], big tile i at boff[i]
    std::vector<int64_t> poff(static_cast<size_t>(n) + 1), boff(static_cast<size_t>(n) + 1);
    for (int64_t i = 0; i < n; ++i) {
        poff[i + 1] = poff[i] + npc[i];
        boff[i + 1] = boff[i] + (npc[i] > 0 ? 0 : 1);
    }
    out.pieces.resize(static_cast<size_t>(poff[n]));
    out.big.resize(static_cast<size_t>(boff[n]));
    std::atomic<bool> off_path{false};
    parallel_for(n, 1 << 14, [&](int64_t a, int64_t b) {
        for (int64_t i = a; i < b; ++i) {
            if (npc[i] == 0) {
                out.big[boff[i]] = list[i];
            } else if (cut_pieces(list[i], es, out.pieces.data() + poff[i]) < 0) {
                off_path = true;
            }
        }
    });
    if (off_path) {  // not expected: keep every small tile whole
        out.pieces.clear();
        out.big = std::move(list);
        return out;
    }
    // groups in list order: at most `cap` pieces of one problem
    auto make_groups = [&](int cap, std::vector<uint32_t> &g) {
        int in_group = 0, group_prob = -1;
        for (size_t k = 0; k < out.pieces.size(); ++k) {
            if (in_group == cap || out.pieces[k].prob != group_prob || g.empty()) {
                g.push_back(static_cast<uint32_t>(k));
                in_group = 0;
                group_prob = out.pieces[k].prob;
            }
            ++in_group;
        }
        if (!g.empty()) g.push_back(static_cast<uint32_t>(out.pieces.size()));
    };
    make_groups(group_pieces(es), out.groups);
    make_groups(group_pieces_a(es, cplx), out.groups_a);
    return out;
}

bool aligned16(uint64_t addr, int64_t ld_bytes) { return ((addr | static_cast<uint64_t>(ld_bytes)) & 15) == 0; }

// The tile (rt, ct) of a problem in the kernel's canonical frame (x = A's
// contiguous axis): source and target addresses of element (0, 0), strides,
// extents, and whether source and target runs lie on different axes.
TileDesc direct_tile(const ProblemHost &ph, const AxisTile &rt, const AxisTile &ct, int es, int prob) {
    const DevBlock &dA = ph.A->blocks[static_cast<size_t>(rt.a_blk) * ph.A->nbc + ct.a_blk];
    const bool tr = ph.op != COSTA_OP_N;
    const DevBlock &dB = tr ? ph.B->blocks[static_cast<size_t>(ct.b_blk) * ph.B->nbc + rt.b_blk]
                            : ph.B->blocks[static_cast<size_t>(rt.b_blk) * ph.B->nbc + ct.b_blk];
    const bool b_col = dB.order == COSTA_COL_MAJOR;
    const int64_t rb = tr ? ct.b_off : rt.b_off, cb = tr ? rt.b_off : ct.b_off;
    const bool src_fast_i = tr ? !b_col : b_col;  // source runs along A's rows
    const bool a_col = dA.order == COSTA_COL_MAJOR;
    TileDesc d;
    d.src = dB.ptr + static_cast<uint64_t>((b_col ? rb + cb * dB.ld : rb * dB.ld + cb) * es);
    d.dst = dA.ptr + static_cast<uint64_t>(
                         (a_col ? rt.a_off + static_cast<int64_t>(ct.a_off) * dA.ld
                                : static_cast<int64_t>(rt.a_off) * dA.ld + ct.a_off) * es);
    d.sld = dB.ld;
    d.dld = dA.ld;
    d.nx = static_cast<uint16_t>(a_col ? rt.len : ct.len);
    d.ny = static_cast<uint16_t>(a_col ? ct.len : rt.len);
    d.prob = static_cast<uint16_t>(prob);
    d.flags = 0;
    if (a_col != src_fast_i) d.flags |= TF_TRANSPOSE;
    if (ph.op == COSTA_OP_C) d.flags |= TF_CONJ;
    return d;
}

// Sets TF_FAST when every run is whole 16-byte chunks on both sides.
void set_fast(TileDesc &d, int es) {
    const int vec = 16 / es;
    const bool tr = (d.flags & TF_TRANSPOSE) != 0;
    const int src_run = tr ? d.ny : d.nx;
    const bool fast = aligned16(d.dst, static_cast<int64_t>(d.dld) * es) &&
                      aligned16(d.src, static_cast<int64_t>(d.sld) * es) && d.nx % vec == 0 &&
                      src_run % vec == 0;
    d.flags = static_cast<uint16_t>(fast ? (d.flags | TF_FAST) : (d.flags & ~TF_FAST));
}

// Visits the tiles of a problem in super-tiles of k x k pieces,
// row pieces fastest inside each: the tiles that warps work on at the same
// time then cover compact regions of A and of B (runs of kSuper tiles along
// both axes) instead of one band of rows across every column.
// Default k: 16 for 16-byte elements (16 x 16 tiles), 8 otherwise (measured
// on GB300).  The environment variable COSTA_SUPER_TILE (1..64) overrides it,
// for tuning.
int super_tile(int esize) {
    static const int env = [] {
        const char *e = std::getenv("COSTA_SUPER_TILE");
        const int v = e ? std::atoi(e) : 0;
        return v >= 1 && v <= 64 ? v : 0;
    }();
    return env ? env : (esize == 16 ? 16 : 8);
}


// Tile order in the target's own storage: each target buffer is walked in
// strips of kLocalStrip tiles across its non-contiguous axis, each strip
// down the buffer's contiguous axis, so that concurrent tiles form long
// contiguous runs of target memory (which is read and written; for a
// transposed problem the source tiles read at the same time are scattered
// whatever the order).  Measured on GB300, 8192^2 unless noted, GB/s:
//  - 8- and 16-byte elements, every op: +6.6% on 16384^2 c128 (C), +2% on
//    f64 (T); op = N: c128 copy BC64 -> BC128 5960 -> 6704, BC128 -> BC32
//    6069 -> 6693, BC32 -> BC256 5962 -> 6350, f64 +1 to +4%, c64 0 to
//    +1.5%;
//  - 4-byte elements: no gain on aligned layouts (32 x 32 f32 tiles; c4
//    -0.3%, f32 N BC16 -> BC64 -20%) and a loss when only the source is
//    misaligned (B's ld odd: 5350 -> 4786), but +7 to +9% when most of the
//    target runs are misaligned and op != N (f32 T copy, A's ld = 1 mod 4:
//    4305 -> 4696; both lds odd 4371 -> 4678; BC50 -> BC75 +2%), where
//    neighbouring tiles share the partial sectors at their ends.
// The environment variable COSTA_TILE_ORDER (global | local) overrides the
// rule, for tuning.
constexpr int kLocalStrip = 2;

bool use_local_order(const ProblemHost &ph, const TileDesc *tiles, size_t n) {
    static const int env = [] {
        const char *e = std::getenv("COSTA_TILE_ORDER");
        if (!e) return -1;
        if (std::strcmp(e, "global") == 0) return 0;
        if (std::strcmp(e, "local") == 0) return 1;
        return -1;
    }();
    if (env >= 0) return env == 1;
    const int es = esize_of(ph.A->dt);
    if (es >= 8) return true;
    return ph.op != COSTA_OP_N && mostly_misaligned(tiles, n, es, true);
}

// Stable LSD radix sort of (key, index) pairs by key, 11 bits per pass (the
// counts and the scatter targets stay in cache); passes stop at the highest
// bit in which two keys differ, and a pass whose digit is equal for every
// key is skipped.
void radix_sort_pairs(std::vector<std::pair<uint64_t, uint32_t>> &v) {
    constexpr int kBits = 11, kBuckets = 1 << kBits;
    std::vector<std::pair<uint64_t, uint32_t>> tmp(v.size());
    std::vector<size_t> count(kBuckets + 1);
    uint64_t lo = ~uint64_t(0), hi = 0;
    for (const auto &e : v) {
        lo = std::min(lo, e.first);
        hi = std::max(hi, e.first);
    }
    for (int shift = 0; shift < 64; shift += kBits) {
        if (((lo ^ hi) >> shift) == 0) break;  // keys agree on every higher bit
        std::fill(count.begin(), count.end(), size_t(0));
        for (const auto &e : v) ++count[((e.first >> shift) & (kBuckets - 1)) + 1];
        bool uniform = false;
        for (int d = 1; d <= kBuckets; ++d)
            if (count[d] == v.size()) uniform = true;
        if (uniform) continue;
        for (int d = 1; d <= kBuckets; ++d) count[d] += count[d - 1];
        for (const auto &e : v) tmp[count[(e.first >> shift) & (kBuckets - 1)]++] = e;
        v.swap(tmp);
    }
}

// Reorders tiles [first, last) (one problem) into the target-local order.
// Tiles are grouped by target stride; within a group an element's local
// coordinates are taken from its offset to the group's lowest target
// address: y = offset / stride (the non-contiguous axis), then strips of
// kLocalStrip * ts along y, ordered by address inside each strip.
void order_tiles_local(std::vector<TileDesc> &list, size_t first, size_t last, int es, int ts) {
    const size_t n = last - first;
    if (n < 2) return;
    std::vector<std::pair<int32_t, uint64_t>> groups;  // (stride, lowest target address)
    std::vector<uint32_t> gid(n);
    for (size_t i = 0; i < n; ++i) {
        const TileDesc &d = list[first + i];
        size_t g = 0;
        while (g < groups.size() && groups[g].first != d.dld) ++g;
        if (g == groups.size()) groups.emplace_back(d.dld, d.dst);
        else groups[g].second = std::min(groups[g].second, d.dst);
        gid[i] = static_cast<uint32_t>(g);
    }
    const uint64_t strip_elems = static_cast<uint64_t>(kLocalStrip) * static_cast<uint64_t>(ts);
    int es_shift = 0;
    while ((1 << es_shift) < es) ++es_shift;
    std::vector<std::pair<uint64_t, uint32_t>> keys(n);
    std::vector<uint64_t> off(n);
    parallel_for(static_cast<int64_t>(n), 1 << 15, [&](int64_t a, int64_t b) {
        for (int64_t i = a; i < b; ++i) {
            const TileDesc &d = list[first + static_cast<size_t>(i)];
            off[i] = (d.dst - groups[gid[i]].second) >> es_shift;
            keys[i] = {off[i] / (static_cast<uint64_t>(d.dld) * strip_elems), static_cast<uint32_t>(i)};
        }
    });
    uint64_t max_strip = 0;
    for (const auto &k : keys) max_strip = std::max(max_strip, k.first);
    // key = group * (max_strip + 1) + strip, so that the sort needs only the
    // bits the keys span
    const uint64_t span = max_strip + 1;
    if (groups.size() > 1 && span <= ~uint64_t(0) / groups.size())
        for (size_t i = 0; i < n; ++i) keys[i].first += gid[keys[i].second] * span;
    radix_sort_pairs(keys);
    // inside each strip, by target address
    std::vector<size_t> runs;  // starts of the runs of equal keys, then n
    for (size_t a = 0; a < n; ++a)
        if (a == 0 || keys[a].first != keys[a - 1].first) runs.push_back(a);
    runs.push_back(n);
    parallel_for(static_cast<int64_t>(runs.size()) - 1, std::max<int64_t>(256, (1 << 15) * static_cast<int64_t>(runs.size()) / std::max<int64_t>(1, static_cast<int64_t>(n))), [&](int64_t r0, int64_t r1) {
        for (int64_t r = r0; r < r1; ++r)
            std::sort(keys.begin() + static_cast<std::ptrdiff_t>(runs[r]),
                      keys.begin() + static_cast<std::ptrdiff_t>(runs[r + 1]),
                      [&](const std::pair<uint64_t, uint32_t> &x, const std::pair<uint64_t, uint32_t> &y) {
                          return off[x.second] < off[y.second];
                      });
    });
    std::vector<TileDesc> tmp(n);
    parallel_for(static_cast<int64_t>(n), 1 << 15, [&](int64_t a, int64_t b) {
        for (int64_t k = a; k < b; ++k) tmp[k] = list[first + keys[k].second];
    });
    std::copy(tmp.begin(), tmp.end(), list.begin() + static_cast<std::ptrdiff_t>(first));
}

// Appends the direct tiles of problem `prob` in the kernel's order.
void append_direct_tiles(const ProblemHost &ph, int prob, int es, int ts, std::vector<TileDesc> &list) {
    const size_t first = list.size();
    // the order of for_each_tile, built in parallel over bands of kSuper row
    // pieces: band su holds the tiles [su * nv, (su + band rows) * nv)
    const int kSuper = super_tile(es);
    const int64_t nu = static_cast<int64_t>(ph.rows.tiles.size()), nv = static_cast<int64_t>(ph.cols.tiles.size());
    list.resize(first + static_cast<size_t>(nu * nv));
    TileDesc *out = list.data() + first;
    const int64_t band_tiles = std::max<int64_t>(1, int64_t(kSuper) * nv);
    parallel_for((nu + kSuper - 1) / kSuper, std::max<int64_t>(1, (1 << 15) / band_tiles), [&](int64_t b0, int64_t b1) {
        for (int64_t band = b0; band < b1; ++band) {
            const int64_t su = band * kSuper, ue = std::min<int64_t>(su + kSuper, nu);
            TileDesc *o = out + su * nv;
            for (int64_t sv = 0; sv < nv; sv += kSuper)
                for (int64_t v = sv; v < std::min<int64_t>(sv + kSuper, nv); ++v)
                    for (int64_t u = su; u < ue; ++u) {
                        TileDesc d = direct_tile(ph, ph.rows.tiles[u], ph.cols.tiles[v], es, prob);
                        set_fast(d, es);
                        *o++ = d;
                    }
        }
    });
    if (!use_local_order(ph, list.data() + first, list.size() - first)) return;
    // a target whose tiles are each one contiguous run gains nothing
    bool contiguous = true;
    for (size_t i = first; i < list.size() && contiguous; ++i) contiguous = list[i].nx == list[i].dld;
    if (!contiguous) order_tiles_local(list, first, list.size(), es, ts);
}

}  // namespace costa
