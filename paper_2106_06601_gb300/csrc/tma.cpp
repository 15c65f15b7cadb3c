// TMA staging of the tile kernel's source tiles (cp.async.bulk.tensor), an
// alternative to per-lane 16-byte cp.async copies: by default for the f64
// general-beta kind (tma_policy_kinds), for every kind with COSTA_TMA=1,
// for none with COSTA_TMA=0.  A plan's TMA lists are built by the first
// call of a kind that uses them (costa.cpp, ensure_tma).
//
// A tensor map describes one 2-D surface of bytes: an allocation of device
// memory viewed as columns of ld_bytes (a block's leading dimension times
// the element size), so every block with that leading dimension inside that
// allocation is a window of the map.  A block-cyclic matrix held in one
// allocation with one local leading dimension for all ranks (a ScaLAPACK
// local matrix per rank, or all ranks in one arena) needs a single map.
// Maps are byte maps (UINT8) with 128-byte swizzling; a box is 128 bytes of
// a run (the inner dimension) by 16 runs.  Loads stay inside the allocation
// (the map's extent is the allocation's, from the driver), so nothing
// outside the caller's memory is read.
//
// A tile qualifies when it is aligned (vector path), has 16 or 32 source
// runs, a run of a whole number of 128-byte boxes, and its source lies in a
// surface that has, or can still get, one of the launch's kMaxTmaMaps maps.
// Its descriptor then carries the box coordinates of its source's (0, 0)
// element: src = (y << 32) | x (x in bytes along the run, y in runs), and
// sld = the map's index.
#include <cuda.h>  // CUtensorMap and its enums; the entry points come from the runtime
#include <cuda_runtime_api.h>

#include <cstdint>
#include <cstdlib>
#include <cstring>
#include <vector>

#include "plan_lists.h"

#ifndef COSTA_TMA_L2
#define COSTA_TMA_L2 CU_TENSOR_MAP_L2_PROMOTION_L2_256B
#endif

namespace costa {

int tma_mode() {
    static const int mode = [] {
        const char *e = std::getenv("COSTA_TMA");
        if (!e) return -1;
        return std::atoi(e) == 1 ? 1 : 0;
    }();
    return mode;
}

// Which kinds take the TMA tiles of a list.  Measured on GB300 (same box,
// 8192^2 f64, GB/s, cp.async -> TMA): the axpby kind with a general beta
// (-0.3, 0.7) 5381 -> 6120 (T, BC64 -> BC128), 5357 -> 6042 (N), 5375 ->
// 6114 (BC32 -> BC256), 5360 -> 6119 (targets of contiguous 16-row
// panels); the cp.async kernel at the TMA instance's occupancy (4 blocks
// without look-ahead) gets only 5682-5701 of that.  Every other kind loses
// with TMA: beta = +-2^k 6397 -> 6198 (c2 6399 -> 6199, c5 6786 -> 6550,
// c5b 6596 -> 6023), copy -5 to -8%, scale -0.2 to -1%, every c64 kind
// -0.5 to -9%, c128 copy (c3) -17%, f32 (c4) -2%.  So only the f64 general
// axpby kind uses it (on its list, the aligned 32 x 32 tiles).
uint32_t tma_policy_kinds(const std::vector<TileDesc> &list, int es, bool cplx, bool halves_list) {
    if (tma_mode() == 0 || list.empty()) return 0;
    if (tma_mode() == 1) return ~0u;
    return (es == 8 && !cplx && !halves_list) ? (1u << K_AXPBY) : 0u;
}

namespace {

using EncodeFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                              const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                              CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
using AttrFn = CUresult (*)(void *, CUpointer_attribute, CUdeviceptr);

template <typename F> F driver_entry(const char *name) {
    void *f = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion(name, &f, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess) {
        cudaGetLastError();
        return nullptr;
    }
    return reinterpret_cast<F>(f);
}

struct Range {
    uint64_t lo, hi;
};

// The allocation holding p, from the driver; false if unknown.
bool allocation_of(uint64_t p, std::vector<Range> &known, Range &out) {
    for (const Range &r : known)
        if (p >= r.lo && p < r.hi) {
            out = r;
            return true;
        }
    static const AttrFn attr = driver_entry<AttrFn>("cuPointerGetAttribute");
    if (!attr) return false;
    CUdeviceptr start = 0;
    size_t size = 0;
    if (attr(&start, CU_POINTER_ATTRIBUTE_RANGE_START_ADDR, static_cast<CUdeviceptr>(p)) != CUDA_SUCCESS ||
        attr(&size, CU_POINTER_ATTRIBUTE_RANGE_SIZE, static_cast<CUdeviceptr>(p)) != CUDA_SUCCESS || size == 0)
        return false;
    out = {static_cast<uint64_t>(start), static_cast<uint64_t>(start) + size};
    if (p < out.lo || p >= out.hi) return false;
    known.push_back(out);
    return true;
}

}  // namespace

void split_tma(std::vector<TileDesc> &list, std::vector<TileDesc> &tma, std::vector<TmaMap> &maps,
               std::vector<uint64_t> &keys, int es) {
    static const EncodeFn encode = driver_entry<EncodeFn>("cuTensorMapEncodeTiled");
    tma.clear();
    if (!encode || list.empty()) return;
    std::vector<Range> known;
    std::vector<TileDesc> rest;
    rest.reserve(list.size());
    for (const TileDesc &d : list) {
        const bool tr = (d.flags & TF_TRANSPOSE) != 0;
        const int runs = tr ? d.nx : d.ny, run_len = tr ? d.ny : d.nx;
        const uint64_t ldb = static_cast<uint64_t>(d.sld) * es, run_bytes = static_cast<uint64_t>(run_len) * es;
        Range r{};
        bool ok = (d.flags & TF_FAST) && (runs == 16 || runs == 32) && run_bytes % 128 == 0 && ldb % 16 == 0 &&
                  ldb <= (uint64_t(1) << 31) && d.src % 16 == 0 && allocation_of(d.src, known, r) && r.lo % 16 == 0;
        uint64_t x = 0, y = 0, ncols = 0;
        int map = -1;
        if (ok) {
            x = (d.src - r.lo) % ldb;
            y = (d.src - r.lo) / ldb;
            ncols = std::min<uint64_t>((r.hi - r.lo) / ldb, uint64_t(1) << 31);
            ok = x % 16 == 0 && x + run_bytes <= ldb && y + runs <= ncols;
        }
        if (ok) {
            for (size_t k = 0; k < maps.size(); ++k)
                if (keys[3 * k] == r.lo && keys[3 * k + 1] == r.hi && keys[3 * k + 2] == ldb) map = static_cast<int>(k);
            if (map < 0 && static_cast<int>(maps.size()) < kMaxTmaMaps) {
                CUtensorMap m;
                const cuuint64_t dims[2] = {ldb, ncols};
                const cuuint64_t strides[1] = {ldb};
                const cuuint32_t box[2] = {128, 16};
                const cuuint32_t estr[2] = {1, 1};
                if (encode(&m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, reinterpret_cast<void *>(r.lo), dims, strides, box,
                           estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                           static_cast<CUtensorMapL2promotion>(COSTA_TMA_L2), CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS) {
                    static_assert(sizeof(CUtensorMap) == sizeof(TmaMap), "tensor map size");
                    TmaMap t;
                    std::memcpy(&t, &m, sizeof t);
                    maps.push_back(t);
                    keys.push_back(r.lo);
                    keys.push_back(r.hi);
                    keys.push_back(ldb);
                    map = static_cast<int>(maps.size()) - 1;
                }
            }
            ok = map >= 0;
        }
        if (!ok) {
            rest.push_back(d);
            continue;
        }
        TileDesc t = d;
        t.src = (y << 32) | x;
        t.sld = map;
        tma.push_back(t);
    }
    list.swap(rest);
}

}  // namespace costa
