// Device tile lists of a plan and their launch, shared by the planner of
// the single-GPU transform (costa.cpp) and the multi-GPU exchange
// (exchange.cpp).  Host code only.
#pragma once

#include <algorithm>
#include <cstring>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "costa_internal.h"
#include "tiles.h"

namespace costa {

// Device copies of a split list inside a plan's arena.
struct DevList {
    const TileDesc *tiles = nullptr;
    int64_t ntiles = 0;
    const TileDesc *mtiles = nullptr;
    int64_t nmtiles = 0;
    const TileDesc *pieces = nullptr;
    const uint32_t *groups = nullptr;
    int64_t ngroups = 0;
    const uint32_t *groups_a = nullptr;  // the groups of the kinds that read A
    int64_t ngroups_a = 0;
    // TMA staging: the kinds in tma_kinds (bit per K_*) run the aligned
    // tiles as rtiles (cp.async) + ttiles (TMA) instead of `tiles`
    const TileDesc *rtiles = nullptr;
    int64_t nrtiles = 0;
    const TileDesc *ttiles = nullptr;
    int64_t nttiles = 0;
    uint32_t tma_kinds = 0;
    bool empty() const { return ntiles == 0 && nmtiles == 0 && ngroups == 0; }
};

struct SplitOffsets {
    size_t tiles, mtiles, pieces, groups, groups_a;
};

// One device allocation holding all tables of a plan, built on the host
// with 256-byte aligned sections and copied once.
struct Arena {
    std::vector<char> host;
    size_t add(const void *p, size_t bytes) {
        const size_t off = (host.size() + 255) & ~size_t(255);
        host.resize(off + std::max<size_t>(bytes, 1));
        if (bytes) std::memcpy(host.data() + off, p, bytes);
        return off;
    }
    template <typename V> size_t add_vec(const std::vector<V> &v) {
        return add(v.data(), v.size() * sizeof(V));
    }
    SplitOffsets add_split(const SplitList &l) {
        return {add_vec(l.big), add_vec(l.mis), add_vec(l.pieces), add_vec(l.groups), add_vec(l.groups_a)};
    }
};

inline DevList resolve(const char *dbase, const SplitOffsets &o, const SplitList &l) {
    DevList d;
    d.tiles = reinterpret_cast<const TileDesc *>(dbase + o.tiles);
    d.ntiles = static_cast<int64_t>(l.big.size());
    d.mtiles = reinterpret_cast<const TileDesc *>(dbase + o.mtiles);
    d.nmtiles = static_cast<int64_t>(l.mis.size());
    d.pieces = reinterpret_cast<const TileDesc *>(dbase + o.pieces);
    d.groups = reinterpret_cast<const uint32_t *>(dbase + o.groups);
    d.ngroups = l.ngroups();
    d.groups_a = reinterpret_cast<const uint32_t *>(dbase + o.groups_a);
    d.ngroups_a = l.ngroups_a();
    return d;
}


// Every tile of a list fits the kernel's tile extent along both axes.
costa_status check_extents(const std::vector<TileDesc> &list, int es, const char *what);

// Every nonempty block of a layout whose owner r has place[r] == g lies in
// memory the current device `dev` can address (the rule of a single-GPU
// transform, applied to the blocks of the ranks on one GPU).
costa_status check_access_on(costa_layout_s *L, int dev, const char *which, const int *place, int g);

// TMA staging of source tiles (COSTA_TMA=1; see tma.cpp): moves the tiles
// of `list` that qualify into `tma`, converted to map coordinates, adding at
// most kMaxTmaMaps maps to `maps`.  Host code; queries the driver for
// allocation ranges.
// COSTA_TMA: unset = the measured policy (the f64 axpby kind with a general
// beta; see tma.cpp), 0 = never, 1 = every kind and type (for A/B
// measurements).
int tma_mode();
uint32_t tma_policy_kinds(const std::vector<TileDesc> &list, int es, bool cplx, bool halves_list);
void split_tma(std::vector<TileDesc> &list, std::vector<TileDesc> &tma, std::vector<TmaMap> &maps,
               std::vector<uint64_t> &keys, int es);

// One element type's scalars alpha[index], beta[index] read from host arrays
// of that type, with the flags that choose the combine kind.
void read_scalar(int dt, const void *p, int index, double out[2]);
Scalars make_scalars(int dt, const void *alpha, const void *beta, int index);

// Launches the remap kernel over a split tile list, once per combine kind
// set in `kinds`: the kinds that run on x-halves take `halves` (when not
// null) for their full-size tiles, and the kinds that read A take the
// small pieces' groups sized for them.
cudaError_t launch_split(const RemapLaunch &base, const DevList &list, const DevList *halves, int esize,
                         const bool (&kinds)[K_NKINDS], cudaStream_t stream);

// An NVTX range over a scope (plan building, the volume kernel, relabeling,
// message and exchange plans, the enqueue of a transform, the exchange's
// phases), visible in Nsight tools; without a tool attached the calls do
// nothing.
struct Trace {
    explicit Trace(const char *name) { nvtxRangePushA(name); }
    ~Trace() { nvtxRangePop(); }
    Trace(const Trace &) = delete;
    Trace &operator=(const Trace &) = delete;
};

// Host log on stderr, lines prefixed "[costa] ": COSTA_LOG=1 logs plans
// (sizes, tiles, times, volumes), relabelings and exchange plans; 2 also
// every transform call.  Off (0) by default.
int log_level();
void log_msg(int level, const char *fmt, ...) __attribute__((format(printf, 2, 3)));

}  // namespace costa
