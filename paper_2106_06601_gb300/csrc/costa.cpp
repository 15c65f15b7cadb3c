// Host side of the library: layout descriptors (Sec. 5 "Matrix Layout",
// Sec. 6 Fig. 1), the grid overlay and tile lists (Sec. 5 "Grid Overlay",
// Alg. 2), the volume / relabeling plan (Alg. 1, Thm. 1), the message-mode
// package offsets (Sec. 6), and the C entry points declared in
// include/costa_gb300.h.
#include <algorithm>
#include <atomic>
#include <chrono>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <map>
#include <memory>
#include <mutex>
#include <string>
#include <thread>
#include <vector>

#include <cuda_runtime_api.h>

#include "costa_internal.h"
#include "fxdot.h"
#include "plan_lists.h"
#include "tiles.h"

namespace costa {

int64_t assign_min(int n, const std::vector<int64_t> &cost, std::vector<int> &row_to_col,
                   std::vector<int64_t> *u_out, std::vector<int64_t> *v_out);
int64_t greedy_max(int P, const int64_t *V, std::vector<int> &sigma);
double assign_min_f(int n, const std::vector<double> &cost, std::vector<int> &row_to_col);
int64_t assign_max_sparse(int P, const int64_t *V, std::vector<int> &sigma);

namespace {

thread_local std::string g_err;
std::atomic<uint64_t> g_next_id{1};

costa_status fail(costa_status s, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_err = buf;
    return s;
}

costa_status cuda_fail(cudaError_t e, const char *what) {
    return fail(COSTA_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

double ms_since(std::chrono::steady_clock::time_point t0) {
    return std::chrono::duration<double, std::milli>(std::chrono::steady_clock::now() - t0).count();
}

struct MessageData {
    bool built = false;
    void *d_mem = nullptr;       // pack, local and unpack tile lists
    DevList pack, local, unpack;
    DevList local_halves, unpack_halves;  // local and unpack with x-halves (see use_halves)
    void *d_staging = nullptr;
    int64_t staging_bytes = 0;
};

struct Plan {
    int device = 0;
    int dtype = 0, esize = 0, P = 0, ts = 32;
    std::vector<ProblemHost> probs;
    void *d_mem = nullptr;
    DevList direct;                     // the direct list
    DevList direct_halves;              // the same with its full aligned tiles in x-halves (4- and 8-byte types)
    Scalars *d_scalars = nullptr;
    std::vector<Scalars> cached_scalars;
    std::vector<TmaMap> tma_maps;       // tensor maps of the TMA-staged tiles
    unsigned int *d_err = nullptr;      // TMA waits that gave up
    // TMA staging (tma.cpp): the kinds that would use it, per list; the
    // lists are built by the first call of such a kind (ensure_tma)
    uint32_t tma_kinds_big = 0, tma_kinds_halves = 0;
    bool tma_built = false;
    void *d_tma = nullptr;
    int64_t total_tiles = 0, total_cells = 0;
    std::vector<int64_t> V;      // P * P, V[p * P + q]
    bool sigma_done = false;
    std::vector<int> sigma;      // optimal relabeling
    costa_plan_stats stats{};
    MessageData msg[2];          // [relabel]
    // Calls that use the plan's device scratch (message mode's staging, the
    // per-problem scalars of a batch) run one after another in call order:
    // a call on another stream than the previous such call first makes its
    // stream wait for that call's completion event.
    cudaEvent_t scratch_done = nullptr;
    cudaStream_t scratch_stream = nullptr;
    bool scratch_used = false;

    ~Plan() {
        for (auto &m : msg) {
            if (m.d_mem) cudaFree(m.d_mem);
            if (m.d_staging) cudaFree(m.d_staging);
        }
        if (d_mem) cudaFree(d_mem);
        if (d_tma) cudaFree(d_tma);
        if (scratch_done) cudaEventDestroy(scratch_done);
    }
};

// Orders a call that uses `plan`'s device scratch after the previous such
// call (see Plan::scratch_done).  Under stream capture nothing is added:
// the caller orders captured work itself.  `capturing` is set for
// scratch_release.
costa_status scratch_acquire(Plan &plan, cudaStream_t stream, bool &capturing) {
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    cudaError_t ce = cudaStreamIsCapturing(stream, &cs);
    if (ce != cudaSuccess) return cuda_fail(ce, "cudaStreamIsCapturing");
    capturing = cs != cudaStreamCaptureStatusNone;
    if (capturing) return COSTA_OK;
    if (!plan.scratch_done) {
        ce = cudaEventCreateWithFlags(&plan.scratch_done, cudaEventDisableTiming);
        if (ce != cudaSuccess) {
            plan.scratch_done = nullptr;
            return cuda_fail(ce, "cudaEventCreate");
        }
    }
    if (plan.scratch_used && plan.scratch_stream != stream) {
        ce = cudaStreamWaitEvent(stream, plan.scratch_done, 0);
        if (ce != cudaSuccess) return cuda_fail(ce, "cudaStreamWaitEvent");
    }
    return COSTA_OK;
}

// Marks the end of a call that used the plan's scratch on `stream`.
costa_status scratch_release(Plan &plan, cudaStream_t stream, bool capturing) {
    if (capturing) return COSTA_OK;
    cudaError_t ce = cudaEventRecord(plan.scratch_done, stream);
    if (ce != cudaSuccess) return cuda_fail(ce, "cudaEventRecord");
    plan.scratch_used = true;
    plan.scratch_stream = stream;
    return COSTA_OK;
}

std::mutex g_mu;
std::map<std::vector<uint64_t>, std::unique_ptr<Plan>> g_plans;

// Phase timing (costa_phase_timing): CUDA events per device, recorded by
// transform calls around their phases.  Guarded by g_mu.
struct PhaseTimer {
    cudaEvent_t ev[4] = {};
    int nphases = 0;  // phases of the last timed call (0: none yet)
};
std::atomic<bool> g_phase_on{false};
std::map<int, PhaseTimer> g_timers;

// The timer of the current device with its events created, or null.
PhaseTimer *phase_timer(costa_status &st) {
    st = COSTA_OK;
    int dev = 0;
    cudaError_t ce = cudaGetDevice(&dev);
    if (ce != cudaSuccess) {
        st = cuda_fail(ce, "cudaGetDevice");
        return nullptr;
    }
    PhaseTimer &t = g_timers[dev];
    for (cudaEvent_t &e : t.ev) {
        if (e) continue;
        ce = cudaEventCreate(&e);
        if (ce != cudaSuccess) {
            st = cuda_fail(ce, "cudaEventCreate");
            return nullptr;
        }
    }
    return &t;
}

bool plan_uses(const std::vector<uint64_t> &key, uint64_t id) {
    // key = [device, n, (A.id, B.id, op) x n]
    for (size_t i = 2; i + 1 < key.size(); i += 3)
        if (key[i] == id || key[i + 1] == id) return true;
    return false;
}

// ---- relabeling: sigma maximizing sum_q V[sigma(q)][q] ----
// Relabeling solver choice: the sparse method for large P with few nonzero
// volumes (a reshuffle sends each target's data from a few sources), the
// dense Hungarian otherwise.  COSTA_RELABEL_SPARSE_MIN_P sets the smallest P
// that may take the sparse method (default 256; 1 forces it wherever V is
// sparse enough, for tests).
int sparse_min_p() {
    static const int v = [] {
        const char *e = std::getenv("COSTA_RELABEL_SPARSE_MIN_P");
        const int k = e ? std::atoi(e) : 0;
        return k >= 1 ? k : 256;
    }();
    return v;
}

void solve_relabel(int P, const int64_t *V, std::vector<int> &sigma, int64_t &best) {
    int64_t nnz = 0;
    for (size_t k = 0; k < static_cast<size_t>(P) * P; ++k) nnz += V[k] > 0;
    std::vector<int> row_to_col;
    if (P >= sparse_min_p() && nnz * 8 <= static_cast<int64_t>(P) * P) {
        best = assign_max_sparse(P, V, row_to_col);
    } else {
        // rows = target labels q, columns = processes p, cost = -V[p][q]
        std::vector<int64_t> cost(static_cast<size_t>(P) * P);
        for (int q = 0; q < P; ++q)
            for (int p = 0; p < P; ++p) cost[static_cast<size_t>(q) * P + p] = -V[static_cast<size_t>(p) * P + q];
        best = -assign_min(P, cost, row_to_col, nullptr, nullptr);
    }
    int64_t trace = 0;
    for (int q = 0; q < P; ++q) trace += V[static_cast<size_t>(q) * P + q];
    sigma.resize(P);
    if (trace == best) {  // tie rule: keep the identity when it is optimal
        for (int q = 0; q < P; ++q) sigma[q] = q;
    } else {
        for (int q = 0; q < P; ++q) sigma[q] = row_to_col[q];
    }
}

costa_status validate_pair(const costa_layout_s *A, const costa_layout_s *B, int op) {
    if (!A || !B) return fail(COSTA_ERR_INVALID_ARG, "null layout");
    if (op < COSTA_OP_N || op > COSTA_OP_C) return fail(COSTA_ERR_INVALID_ARG, "bad op %d", op);
    if (A->dt != B->dt)
        return fail(COSTA_ERR_DTYPE, "element types differ (A %d, B %d)", A->dt, B->dt);
    if (A->nranks != B->nranks)
        return fail(COSTA_ERR_SHAPE, "rank counts differ (A %d, B %d)", A->nranks, B->nranks);
    const int64_t bm = op == COSTA_OP_N ? B->m : B->n, bn = op == COSTA_OP_N ? B->n : B->m;
    if (A->m != bm || A->n != bn)
        return fail(COSTA_ERR_SHAPE, "A is %lld x %lld but op(B) is %lld x %lld", (long long)A->m,
                    (long long)A->n, (long long)bm, (long long)bn);
    return COSTA_OK;
}

// ---- storage access ----
//
// Every nonempty block's first and last element must lie in one allocation
// the current device can address: its own device memory, managed memory, or
// host memory allocated or registered with CUDA (the kernels then read and
// write it over the host link; with unified addressing the host address
// serves the device too).  Pageable host memory, another device's memory and
// unknown addresses are rejected with COSTA_ERR_LAYOUT before any kernel
// runs.  Allocation ranges come from the driver (one query per allocation,
// then a binary search per block); the result is kept per layout and device.

typedef int (*PointerAttrFn)(void *data, int attribute, unsigned long long ptr);

PointerAttrFn pointer_attr_fn() {
    static PointerAttrFn fn = [] {
        void *f = nullptr;
        cudaDriverEntryPointQueryResult q{};
        if (cudaGetDriverEntryPointByVersion("cuPointerGetAttribute", &f, 12000, cudaEnableDefault, &q) !=
                cudaSuccess ||
            q != cudaDriverEntryPointSuccess) {
            cudaGetLastError();
            f = nullptr;
        }
        return reinterpret_cast<PointerAttrFn>(f);
    }();
    return fn;
}

struct AccessRange {
    uint64_t lo, hi;  // [lo, hi)
};

// The allocation holding `p` if the device `dev` may access it; on failure
// a message in `why`.
bool access_range(uint64_t p, int dev, AccessRange &r, std::string &why) {
    cudaPointerAttributes a{};
    if (cudaPointerGetAttributes(&a, reinterpret_cast<const void *>(p)) != cudaSuccess) {
        cudaGetLastError();
        why = "address unknown to CUDA";
        return false;
    }
    switch (a.type) {
    case cudaMemoryTypeDevice:
        if (a.device != dev) {
            why = "memory of device " + std::to_string(a.device) + ", not of the current device " + std::to_string(dev);
            return false;
        }
        break;
    case cudaMemoryTypeManaged:
        break;
    case cudaMemoryTypeHost:
        if (reinterpret_cast<uint64_t>(a.devicePointer) != p) {
            why = "host memory not mapped at the same address on the device";
            return false;
        }
        break;
    default:
        why = "pageable host memory (allocate it with cudaHostAlloc or register it with cudaHostRegister)";
        return false;
    }
    r.lo = p;
    r.hi = p + 1;
    if (PointerAttrFn fn = pointer_attr_fn()) {
        unsigned long long start = 0;
        size_t size = 0;
        constexpr int kRangeStart = 11, kRangeSize = 12;  // CU_POINTER_ATTRIBUTE_RANGE_START_ADDR / _SIZE
        if (fn(&start, kRangeStart, p) == 0 && fn(&size, kRangeSize, p) == 0 && size > 0 && start <= p &&
            p < start + size) {
            r.lo = start;
            r.hi = start + size;
        }
    }
    return true;
}

// With `place` set, only the blocks whose owner r has place[r] == g are
// checked (the multi-GPU exchange), and the result is not cached.
costa_status check_access_impl(costa_layout_s *L, int dev, const char *which, const int *place, int g) {
    if (!place && L->checked_device == dev) return COSTA_OK;
    const int64_t es = esize_of(L->dt);
    std::vector<AccessRange> known;  // sorted by lo, disjoint
    auto covered = [&](uint64_t a, uint64_t b) {  // [a, b] inside one known range
        auto it = std::upper_bound(known.begin(), known.end(), a,
                                   [](uint64_t v, const AccessRange &r) { return v < r.lo; });
        if (it == known.begin()) return false;
        --it;
        return a >= it->lo && b < it->hi;
    };
    auto add = [&](const AccessRange &r) {
        auto it = std::lower_bound(known.begin(), known.end(), r.lo,
                                   [](const AccessRange &k, uint64_t v) { return k.lo < v; });
        known.insert(it, r);
    };
    for (int i = 0; i < L->nbr; ++i) {
        const int64_t rows = L->R[i + 1] - L->R[i];
        for (int j = 0; j < L->nbc; ++j) {
            const int64_t cols = L->C[j + 1] - L->C[j];
            if (rows == 0 || cols == 0) continue;
            if (place && place[L->owner[static_cast<size_t>(i) * L->nbc + j]] != g) continue;
            const DevBlock &b = L->blocks[static_cast<size_t>(i) * L->nbc + j];
            const int64_t last = b.order == COSTA_COL_MAJOR ? (rows - 1) + (cols - 1) * int64_t(b.ld)
                                                            : (rows - 1) * int64_t(b.ld) + (cols - 1);
            if (!b.ptr)
                return fail(COSTA_ERR_LAYOUT, "%s block (%d, %d) has no storage in this process (null pointer)",
                            which, i, j);
            const uint64_t first = b.ptr, end = b.ptr + static_cast<uint64_t>((last + 1) * es - 1);
            if (covered(first, end)) continue;
            AccessRange r;
            std::string why;
            if (!access_range(first, dev, r, why))
                return fail(COSTA_ERR_LAYOUT, "%s block (%d, %d): %s", which, i, j, why.c_str());
            if (r.hi <= end) {  // no range from the driver, or the block leaves it
                AccessRange r2;
                if (!access_range(end, dev, r2, why))
                    return fail(COSTA_ERR_LAYOUT, "%s block (%d, %d), last element: %s", which, i, j, why.c_str());
                if (r.hi - r.lo > 1 || r2.hi - r2.lo > 1)  // ranges known: the block spans two allocations
                    return fail(COSTA_ERR_LAYOUT, "%s block (%d, %d) spans two allocations", which, i, j);
                continue;  // both ends accessible, no ranges to cache
            }
            add(r);
        }
    }
    if (!place) L->checked_device = dev;
    return COSTA_OK;
}

costa_status check_access(costa_layout_s *L, int dev, const char *which) {
    return check_access_impl(L, dev, which, nullptr, 0);
}

// Builds the overlay, the tile list and the device tables, and runs the
// volume kernel.
costa_status build_plan(int n, const costa_layout *As, const costa_layout *Bs, const costa_op *ops,
                        cudaStream_t stream, std::unique_ptr<Plan> &out) {
    Trace range("costa plan");
    auto t0 = std::chrono::steady_clock::now();
    auto plan = std::make_unique<Plan>();
    cudaError_t ce = cudaGetDevice(&plan->device);
    if (ce != cudaSuccess) return cuda_fail(ce, "cudaGetDevice");
    if (n > 65535) return fail(COSTA_ERR_INVALID_ARG, "batch of %d exceeds 65535 pairs", n);
    for (int k = 0; k < n; ++k) {
        costa_status st = check_access(As[k], plan->device, "A");
        if (st == COSTA_OK) st = check_access(Bs[k], plan->device, "B");
        if (st != COSTA_OK) return st;
    }
    plan->dtype = As[0]->dt;
    plan->esize = esize_of(plan->dtype);
    plan->P = As[0]->nranks;
    plan->ts = tile_extent(plan->esize);
    const int P = plan->P, ts = plan->ts, es = plan->esize;

    Arena arena;
    struct Off { size_t irows, icols, ownA, ownB; };
    std::vector<Off> offs(n);
    int64_t tiles = 0, cells = 0;
    for (int k = 0; k < n; ++k) {
        ProblemHost ph;
        ph.A = As[k];
        ph.B = Bs[k];
        ph.op = ops[k];
        ph.rows = cut_pair_axis(ph.A, ph.B, ph.op, 0, ts);
        ph.cols = cut_pair_axis(ph.A, ph.B, ph.op, 1, ts);
        Off &o = offs[k];
        o.irows = arena.add_vec(ph.rows.intervals);
        o.icols = arena.add_vec(ph.cols.intervals);
        o.ownA = arena.add_vec(ph.A->owner);
        o.ownB = arena.add_vec(ph.B->owner);
        tiles += static_cast<int64_t>(ph.rows.tiles.size()) * static_cast<int64_t>(ph.cols.tiles.size());
        cells += static_cast<int64_t>(ph.rows.intervals.size()) * static_cast<int64_t>(ph.cols.intervals.size());
        plan->probs.push_back(std::move(ph));
    }
    // the direct tile list, in (problem, row piece, column piece) order
    std::vector<TileDesc> list;
    if (n == 1) {
        append_direct_tiles(plan->probs[0], 0, es, ts, list);
    } else {  // a batch: problems in parallel, each into its own range
        std::vector<int64_t> start(static_cast<size_t>(n) + 1, 0);
        for (int k = 0; k < n; ++k)
            start[k + 1] = start[k] + static_cast<int64_t>(plan->probs[k].rows.tiles.size()) *
                                          static_cast<int64_t>(plan->probs[k].cols.tiles.size());
        list.resize(static_cast<size_t>(start[n]));
        parallel_for(n, std::max<int64_t>(1, (int64_t(1) << 15) * n / std::max<int64_t>(1, start[n])),
                     [&](int64_t k0, int64_t k1) {
                         for (int64_t k = k0; k < k1; ++k) {
                             std::vector<TileDesc> part;
                             append_direct_tiles(plan->probs[k], static_cast<int>(k), es, ts, part);
                             std::copy(part.begin(), part.end(), list.begin() + start[k]);
                         }
                     });
    }
    {
        costa_status st = check_extents(list, es, "direct");
        if (st != COSTA_OK) return st;
    }
    const bool cplx = plan->dtype == COSTA_C64 || plan->dtype == COSTA_C128;
    SplitList split = split_small(std::move(list), es, cplx);
    // The aligned tiles also as x-halves (see use_halves), for the kinds
    // that run on them (see launch_list in transform_impl).
    std::vector<char> halve(static_cast<size_t>(n), 0);
    for (int k = 0; k < n; ++k) halve[k] = use_halves(plan->probs[k], es);
    std::vector<TileDesc> halves = split_x_halves(split.big, ts / 2, es, halve);
    const bool had_halves = !halves.empty();
    // TMA staging (tma.cpp): the kinds the policy would give it; their lists
    // are built by the first call of such a kind (ensure_tma)
    plan->tma_kinds_big = tma_policy_kinds(split.big, es, cplx, false);
    plan->tma_kinds_halves = had_halves ? tma_policy_kinds(halves, es, cplx, true) : 0;
    const SplitOffsets off_tiles = arena.add_split(split);
    const size_t off_halves = halves.empty() ? 0 : arena.add_vec(halves);
    const uint32_t zero_word = 0;
    const size_t off_err = arena.add(&zero_word, sizeof zero_word);
    std::vector<VolumeProblemDev> vd(n);
    const size_t off_vd = arena.add(vd.data(), sizeof(VolumeProblemDev) * n);
    std::vector<Scalars> sc(n);
    const size_t off_sc = arena.add(sc.data(), sizeof(Scalars) * n);
    std::vector<unsigned long long> vz(static_cast<size_t>(P) * P, 0ull);
    const size_t off_V = arena.add_vec(vz);

    void *d = nullptr;
    ce = cudaMalloc(&d, arena.host.size());
    if (ce != cudaSuccess) return fail(COSTA_ERR_ALLOC, "cudaMalloc(%zu): %s", arena.host.size(),
                                       cudaGetErrorString(ce));
    plan->d_mem = d;
    char *dbase = static_cast<char *>(d);
    int64_t cell_begin = 0;
    for (int k = 0; k < n; ++k) {
        const ProblemHost &ph = plan->probs[k];
        const Off &o = offs[k];
        VolumeProblemDev &v = vd[k];
        v.rows = reinterpret_cast<const Interval *>(dbase + o.irows);
        v.cols = reinterpret_cast<const Interval *>(dbase + o.icols);
        v.ownerA = reinterpret_cast<const int32_t *>(dbase + o.ownA);
        v.ownerB = reinterpret_cast<const int32_t *>(dbase + o.ownB);
        v.cell_begin = cell_begin;
        v.nr = static_cast<int32_t>(ph.rows.intervals.size());
        v.nc = static_cast<int32_t>(ph.cols.intervals.size());
        v.nbcA = ph.A->nbc;
        v.nbcB = ph.B->nbc;
        v.op = ph.op;
        v.pad = 0;
        cell_begin += static_cast<int64_t>(v.nr) * v.nc;
    }
    std::memcpy(arena.host.data() + off_vd, vd.data(), sizeof(VolumeProblemDev) * n);
    ce = cudaMemcpy(d, arena.host.data(), arena.host.size(), cudaMemcpyHostToDevice);
    if (ce != cudaSuccess) return cuda_fail(ce, "cudaMemcpy(plan tables)");
    plan->direct = resolve(dbase, off_tiles, split);
    plan->direct_halves = plan->direct;
    if (had_halves) {
        plan->direct_halves.tiles = reinterpret_cast<const TileDesc *>(dbase + off_halves);
        plan->direct_halves.ntiles = static_cast<int64_t>(halves.size());
    }
    plan->d_err = reinterpret_cast<unsigned int *>(dbase + off_err);
    plan->d_scalars = reinterpret_cast<Scalars *>(dbase + off_sc);
    plan->total_tiles = tiles;
    plan->total_cells = cells;

    // volume kernel: V[p][q] over the overlay cells
    Trace range_v("costa volume");
    auto tv = std::chrono::steady_clock::now();
    VolumeLaunch vl;
    vl.probs = reinterpret_cast<const VolumeProblemDev *>(dbase + off_vd);
    vl.nprob = n;
    vl.P = P;
    vl.total_cells = cells;
    vl.V = reinterpret_cast<unsigned long long *>(dbase + off_V);
    ce = launch_volume(vl, stream);
    if (ce != cudaSuccess) return cuda_fail(ce, "volume kernel launch");
    plan->V.assign(static_cast<size_t>(P) * P, 0);
    ce = cudaMemcpyAsync(plan->V.data(), vl.V, sizeof(int64_t) * P * P, cudaMemcpyDeviceToHost, stream);
    if (ce != cudaSuccess) return cuda_fail(ce, "cudaMemcpyAsync(V)");
    ce = cudaStreamSynchronize(stream);
    if (ce != cudaSuccess) return cuda_fail(ce, "volume kernel");
    plan->stats.volume_ms = ms_since(tv);

    int64_t total = 0, trace = 0;
    for (int p = 0; p < P; ++p)
        for (int q = 0; q < P; ++q) total += plan->V[static_cast<size_t>(p) * P + q];
    for (int q = 0; q < P; ++q) trace += plan->V[static_cast<size_t>(q) * P + q];
    int64_t want = 0;
    for (int k = 0; k < n; ++k) want += As[k]->m * As[k]->n;
    if (total != want)
        return fail(COSTA_ERR_INTERNAL, "volume check failed: sum V = %lld, expected %lld",
                    (long long)total, (long long)want);
    plan->stats.total_volume = total;
    plan->stats.local_identity = trace;
    plan->stats.local_relabeled = trace;
    plan->stats.n_cells = cells;
    plan->stats.n_tiles = tiles;
    plan->stats.plan_ms = ms_since(t0);
    log_msg(1, "plan: %d pair(s), dtype %d, P = %d, %lld cells, %lld tiles (%lld direct, %lld misaligned, "
               "%lld small pieces), total volume %lld, local %lld; %.2f ms (volume %.2f ms)",
            n, plan->dtype, P, (long long)cells, (long long)tiles, (long long)split.big.size(),
            (long long)split.mis.size(), (long long)split.pieces.size(), (long long)total, (long long)trace,
            plan->stats.plan_ms, plan->stats.volume_ms);
    out = std::move(plan);
    return COSTA_OK;
}

costa_status ensure_sigma(Plan &plan) {
    if (plan.sigma_done) return COSTA_OK;
    Trace trace("costa relabel");
    auto t0 = std::chrono::steady_clock::now();
    int64_t best = 0;
    solve_relabel(plan.P, plan.V.data(), plan.sigma, best);
    plan.stats.relabel_ms = ms_since(t0);
    log_msg(1, "relabel: P = %d, local volume %lld -> %lld of %lld; %.3f ms", plan.P,
            (long long)plan.stats.local_identity, (long long)best, (long long)plan.stats.total_volume,
            plan.stats.relabel_ms);
    plan.stats.local_relabeled = best;
    plan.sigma_done = true;
    return COSTA_OK;
}

// The TMA split of the aligned lists (tma.cpp) for the kinds that use it,
// built by the first call that needs it: the lists come back from the
// device, are split, and go up again in an allocation of their own, with
// synchronous copies.  Plans of other kinds never pay for it.
costa_status ensure_tma(Plan &plan) {
    if (plan.tma_built) return COSTA_OK;
    plan.tma_built = true;
    if (!plan.tma_kinds_big && !plan.tma_kinds_halves) return COSTA_OK;
    Trace trace("costa tma lists");
    const int es = plan.esize;
    const bool halves = plan.direct_halves.tiles != plan.direct.tiles;
    std::vector<TileDesc> big(static_cast<size_t>(plan.direct.ntiles));
    std::vector<TileDesc> hv(halves && plan.tma_kinds_halves ? static_cast<size_t>(plan.direct_halves.ntiles) : 0);
    cudaError_t ce = cudaSuccess;
    if (plan.tma_kinds_big && !big.empty())
        ce = cudaMemcpy(big.data(), plan.direct.tiles, sizeof(TileDesc) * big.size(), cudaMemcpyDeviceToHost);
    if (ce == cudaSuccess && !hv.empty())
        ce = cudaMemcpy(hv.data(), plan.direct_halves.tiles, sizeof(TileDesc) * hv.size(), cudaMemcpyDeviceToHost);
    if (ce != cudaSuccess) return cuda_fail(ce, "cudaMemcpy(tile lists)");
    std::vector<TileDesc> tma_big, tma_hv;
    std::vector<uint64_t> keys;
    if (plan.tma_kinds_big) split_tma(big, tma_big, plan.tma_maps, keys, es);
    if (!hv.empty()) split_tma(hv, tma_hv, plan.tma_maps, keys, es);
    if (tma_big.empty() && tma_hv.empty()) return COSTA_OK;
    Arena arena;
    const size_t o_rb = arena.add_vec(big), o_tb = arena.add_vec(tma_big);
    const size_t o_rh = arena.add_vec(hv), o_th = arena.add_vec(tma_hv);
    ce = cudaMalloc(&plan.d_tma, arena.host.size());
    if (ce != cudaSuccess) {
        plan.d_tma = nullptr;
        return fail(COSTA_ERR_ALLOC, "cudaMalloc(TMA tile lists): %s", cudaGetErrorString(ce));
    }
    ce = cudaMemcpy(plan.d_tma, arena.host.data(), arena.host.size(), cudaMemcpyHostToDevice);
    if (ce != cudaSuccess) return cuda_fail(ce, "cudaMemcpy(TMA tile lists)");
    const char *db = static_cast<const char *>(plan.d_tma);
    if (!tma_big.empty()) {
        DevList &d = plan.direct;
        d.rtiles = reinterpret_cast<const TileDesc *>(db + o_rb);
        d.nrtiles = static_cast<int64_t>(big.size());
        d.ttiles = reinterpret_cast<const TileDesc *>(db + o_tb);
        d.nttiles = static_cast<int64_t>(tma_big.size());
        d.tma_kinds = plan.tma_kinds_big;
    }
    DevList &h = plan.direct_halves;
    if (!halves) {  // the halves list is the direct list
        const DevList tiles_only = h;
        h = plan.direct;
        h.tiles = tiles_only.tiles;
        h.ntiles = tiles_only.ntiles;
    } else if (!tma_hv.empty()) {
        h.rtiles = reinterpret_cast<const TileDesc *>(db + o_rh);
        h.nrtiles = static_cast<int64_t>(hv.size());
        h.ttiles = reinterpret_cast<const TileDesc *>(db + o_th);
        h.nttiles = static_cast<int64_t>(tma_hv.size());
        h.tma_kinds = plan.tma_kinds_halves;
    }
    log_msg(1, "TMA lists: %zu + %zu tiles, %zu map(s)", tma_big.size(), tma_hv.size(), plan.tma_maps.size());
    return COSTA_OK;
}

// Message mode (Alg. 3, Sec. 6): every tile whose source process p differs
// from the process sigma(q) that takes its target label q is "remote" and
// travels through the staging buffer.  Packages are ordered by (p, receiver)
// at the exclusive-scan offsets of their sizes; inside a package the tiles
// keep the tile order.  Each staged tile is dense in the source's element
// order with its leading dimension rounded up to 16 bytes.  Three tile lists
// result: pack (B -> staging), local (B -> A) and unpack (staging -> A).
costa_status ensure_message(Plan &plan, bool relabel) {
    MessageData &m = plan.msg[relabel ? 1 : 0];
    if (m.built) return COSTA_OK;
    Trace trace("costa message plan");
    const int P = plan.P, es = plan.esize;
    std::vector<int> sig(P);
    if (relabel) {
        costa_status s = ensure_sigma(plan);
        if (s != COSTA_OK) return s;
        sig = plan.sigma;
    } else {
        for (int q = 0; q < P; ++q) sig[q] = q;
    }
    const int vec = 16 / es;
    struct Remote { TileDesc d; int32_t pkg; int32_t ld; int64_t size; };
    std::vector<TileDesc> local;
    std::vector<Remote> remote;
    std::vector<int64_t> size(static_cast<size_t>(P) * P, 0);
    for (size_t k = 0; k < plan.probs.size(); ++k) {
        const ProblemHost &ph = plan.probs[k];
        const bool tr = ph.op != COSTA_OP_N;
        for_each_tile(ph, [&](const AxisTile &rt, const AxisTile &ct) {
            {
                TileDesc d = direct_tile(ph, rt, ct, es, static_cast<int>(k));
                const int q = ph.A->owner[static_cast<size_t>(rt.a_blk) * ph.A->nbc + ct.a_blk];
                const size_t bidx = tr ? static_cast<size_t>(ct.b_blk) * ph.B->nbc + rt.b_blk
                                       : static_cast<size_t>(rt.b_blk) * ph.B->nbc + ct.b_blk;
                const int p = ph.B->owner[bidx];
                if (p == sig[q]) {
                    set_fast(d, es);
                    local.push_back(d);
                    return;
                }
                const bool t = (d.flags & TF_TRANSPOSE) != 0;
                const int fast = t ? d.ny : d.nx, other = t ? d.nx : d.ny;  // source frame
                Remote r;
                r.d = d;
                r.pkg = p * P + sig[q];
                r.ld = (fast + vec - 1) / vec * vec;
                r.size = static_cast<int64_t>(r.ld) * other;
                size[static_cast<size_t>(r.pkg)] += r.size;
                remote.push_back(r);
            }
        });
    }
    std::vector<int64_t> base(static_cast<size_t>(P) * P, 0);
    int64_t acc = 0;
    for (size_t k = 0; k < base.size(); ++k) {
        base[k] = acc;
        acc += size[k];
    }
    m.staging_bytes = acc * es;
    if (m.staging_bytes > 0) {
        cudaError_t ce = cudaMalloc(&m.d_staging, static_cast<size_t>(m.staging_bytes));
        if (ce != cudaSuccess)
            return fail(COSTA_ERR_ALLOC, "cudaMalloc(staging %lld B): %s", (long long)m.staging_bytes,
                        cudaGetErrorString(ce));
    }
    const uint64_t stage = reinterpret_cast<uint64_t>(m.d_staging);
    std::vector<TileDesc> pack, unpack;
    pack.reserve(remote.size());
    unpack.reserve(remote.size());
    for (const Remote &r : remote) {
        const int64_t off = base[static_cast<size_t>(r.pkg)];
        base[static_cast<size_t>(r.pkg)] += r.size;
        const uint64_t addr = stage + static_cast<uint64_t>(off * es);
        // pack: an exact copy in the source's frame (x = the source's contiguous axis)
        TileDesc pk = r.d;
        const bool t = (r.d.flags & TF_TRANSPOSE) != 0;
        pk.nx = t ? r.d.ny : r.d.nx;
        pk.ny = t ? r.d.nx : r.d.ny;
        pk.dst = addr;
        pk.dld = r.ld;
        pk.flags = 0;
        set_fast(pk, es);
        pack.push_back(pk);
        // unpack: the direct tile reading the staged copy
        TileDesc up = r.d;
        up.src = addr;
        up.sld = r.ld;
        set_fast(up, es);
        unpack.push_back(up);
    }
    for (const auto &l : {std::make_pair(&pack, "pack"), std::make_pair(&local, "local"),
                          std::make_pair(&unpack, "unpack")}) {
        costa_status st = check_extents(*l.first, es, l.second);
        if (st != COSTA_OK) return st;
    }
    const bool cplx = plan.dtype == COSTA_C64 || plan.dtype == COSTA_C128;
    const SplitList s_pack = split_small(std::move(pack), es, cplx),
                    s_local = split_small(std::move(local), es, cplx),
                    s_unpack = split_small(std::move(unpack), es, cplx);
    std::vector<char> halve(plan.probs.size(), 0);
    for (size_t k = 0; k < plan.probs.size(); ++k) halve[k] = use_halves(plan.probs[k], es);
    const std::vector<TileDesc> h_local = split_x_halves(s_local.big, plan.ts / 2, es, halve),
                                h_unpack = split_x_halves(s_unpack.big, plan.ts / 2, es, halve);
    Arena arena;
    const SplitOffsets o_pack = arena.add_split(s_pack);
    const SplitOffsets o_local = arena.add_split(s_local);
    const SplitOffsets o_unpack = arena.add_split(s_unpack);
    const size_t o_hl = h_local.empty() ? 0 : arena.add_vec(h_local);
    const size_t o_hu = h_unpack.empty() ? 0 : arena.add_vec(h_unpack);
    cudaError_t ce = cudaMalloc(&m.d_mem, arena.host.size());
    if (ce != cudaSuccess) return fail(COSTA_ERR_ALLOC, "cudaMalloc(message tables): %s", cudaGetErrorString(ce));
    ce = cudaMemcpy(m.d_mem, arena.host.data(), arena.host.size(), cudaMemcpyHostToDevice);
    if (ce != cudaSuccess) return cuda_fail(ce, "cudaMemcpy(message tables)");
    const char *db = static_cast<const char *>(m.d_mem);
    m.pack = resolve(db, o_pack, s_pack);
    m.local = resolve(db, o_local, s_local);
    m.unpack = resolve(db, o_unpack, s_unpack);
    m.local_halves = m.local;
    m.unpack_halves = m.unpack;
    if (!h_local.empty()) {
        m.local_halves.tiles = reinterpret_cast<const TileDesc *>(db + o_hl);
        m.local_halves.ntiles = static_cast<int64_t>(h_local.size());
    }
    if (!h_unpack.empty()) {
        m.unpack_halves.tiles = reinterpret_cast<const TileDesc *>(db + o_hu);
        m.unpack_halves.ntiles = static_cast<int64_t>(h_unpack.size());
    }
    m.built = true;
    plan.stats.staging_bytes = m.staging_bytes;
    log_msg(1, "message plan (relabel %d): staging %lld bytes, pack %lld, local %lld, unpack %lld tiles",
            relabel ? 1 : 0, (long long)m.staging_bytes, (long long)(m.pack.ntiles + m.pack.nmtiles),
            (long long)(m.local.ntiles + m.local.nmtiles), (long long)(m.unpack.ntiles + m.unpack.nmtiles));
    return COSTA_OK;
}

costa_status get_plan(int n, const costa_layout *A, const costa_layout *B, const costa_op *ops,
                      cudaStream_t stream, Plan *&out) {
    int dev = 0;
    cudaError_t ce = cudaGetDevice(&dev);
    if (ce != cudaSuccess) return cuda_fail(ce, "cudaGetDevice");
    std::vector<uint64_t> key;
    key.reserve(2 + 3 * static_cast<size_t>(n));
    key.push_back(static_cast<uint64_t>(dev));
    key.push_back(static_cast<uint64_t>(n));
    for (int k = 0; k < n; ++k) {
        key.push_back(A[k]->id);
        key.push_back(B[k]->id);
        key.push_back(static_cast<uint64_t>(ops[k]));
    }
    auto it = g_plans.find(key);
    if (it != g_plans.end()) {
        out = it->second.get();
        return COSTA_OK;
    }
    std::unique_ptr<Plan> plan;
    costa_status s = build_plan(n, A, B, ops, stream, plan);
    if (s != COSTA_OK) return s;
    out = plan.get();
    g_plans.emplace(std::move(key), std::move(plan));
    return COSTA_OK;
}

// Reads one scalar of element type dt at p[index].
bool same_scalars(const Scalars &a, const Scalars &b) { return std::memcmp(&a, &b, sizeof(Scalars)) == 0; }

costa_status transform_impl(int n, const costa_layout *A, const costa_layout *B, const costa_op *ops,
                            const void *alphas, const void *betas, int relabel, int *sigma_out,
                            int mode, void *stream_v) {
    if (n < 1) return fail(COSTA_ERR_INVALID_ARG, "batch size %d < 1", n);
    if (!A || !B || !ops || !alphas || !betas) return fail(COSTA_ERR_INVALID_ARG, "null argument");
    if (mode != COSTA_MODE_DIRECT && mode != COSTA_MODE_MESSAGE)
        return fail(COSTA_ERR_INVALID_ARG, "bad mode %d", mode);
    for (int k = 0; k < n; ++k) {
        costa_status s = validate_pair(A[k], B[k], ops[k]);
        if (s != COSTA_OK) return s;
        if (A[k]->dt != A[0]->dt) return fail(COSTA_ERR_DTYPE, "batch mixes element types");
        if (A[k]->nranks != A[0]->nranks) return fail(COSTA_ERR_SHAPE, "batch mixes rank counts");
    }
    cudaStream_t stream = static_cast<cudaStream_t>(stream_v);
    std::lock_guard<std::mutex> lock(g_mu);
    Plan *plan = nullptr;
    costa_status s = get_plan(n, A, B, ops, stream, plan);
    if (s != COSTA_OK) return s;
    const int P = plan->P;
    if (relabel) {
        s = ensure_sigma(*plan);
        if (s != COSTA_OK) return s;
    }
    if (sigma_out)
        for (int q = 0; q < P; ++q) sigma_out[q] = relabel ? plan->sigma[q] : q;
    PhaseTimer *timer = nullptr;
    if (g_phase_on.load()) {
        timer = phase_timer(s);
        if (!timer) return s;
        timer->nphases = 0;
    }
    if (plan->total_tiles == 0) return COSTA_OK;
    Trace trace("costa transform");
    log_msg(2, "transform: %d pair(s), %s mode, relabel %d, stream %p", n,
            mode == COSTA_MODE_DIRECT ? "direct" : "message", relabel ? 1 : 0, static_cast<void *>(stream));
    // event k marks the end of phase k (event 0: the start)
    auto mark = [&](int k) -> cudaError_t { return timer ? cudaEventRecord(timer->ev[k], stream) : cudaSuccess; };

    RemapLaunch L{};
    L.dtype = plan->dtype;
    L.s = make_scalars(plan->dtype, alphas, betas, 0);
    L.per_problem = nullptr;
    bool uniform = true;
    std::vector<Scalars> sc(n);
    for (int k = 0; k < n; ++k) {
        sc[k] = make_scalars(plan->dtype, alphas, betas, k);
        if (!same_scalars(sc[k], sc[0])) uniform = false;
    }
    // one launch per combine kind present in the batch
    bool kinds[K_NKINDS] = {};
    for (int k = 0; k < n; ++k) kinds[kind_of(sc[k].flags)] = true;
    if (!plan->tma_built && mode == COSTA_MODE_DIRECT) {
        bool want = false;
        for (int kind = 0; kind < K_NKINDS; ++kind)
            want |= kinds[kind] && (((plan->tma_kinds_big | plan->tma_kinds_halves) >> kind) & 1u);
        cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
        if (want && cudaStreamIsCapturing(stream, &cs) == cudaSuccess && cs == cudaStreamCaptureStatusNone) {
            s = ensure_tma(*plan);  // under capture the cp.async lists serve
            if (s != COSTA_OK) return s;
        }
    }
    // the calls that use the plan's scratch are ordered (Plan::scratch_done)
    const bool uses_scratch = !uniform || mode == COSTA_MODE_MESSAGE;
    bool capturing = false;
    if (uses_scratch) {
        s = scratch_acquire(*plan, stream, capturing);
        if (s != COSTA_OK) return s;
    }
    auto done = [&](costa_status st) -> costa_status {
        if (st != COSTA_OK || !uses_scratch) return st;
        return scratch_release(*plan, stream, capturing);
    };
    if (!uniform) {
        bool same = plan->cached_scalars.size() == sc.size();
        for (int k = 0; same && k < n; ++k) same = same_scalars(sc[k], plan->cached_scalars[k]);
        if (!same) {
            // pageable source: the copy is staged before the call returns, and
            // stream order places it after earlier kernels of this stream
            cudaError_t ce = cudaMemcpyAsync(plan->d_scalars, sc.data(), sizeof(Scalars) * n,
                                             cudaMemcpyHostToDevice, stream);
            if (ce != cudaSuccess) {
                plan->cached_scalars.clear();
                return cuda_fail(ce, "cudaMemcpyAsync(scalars)");
            }
            plan->cached_scalars = sc;
        }
        L.per_problem = plan->d_scalars;
    }
    TmaLists tma_base{};  // the plan's tensor maps and error word (launch_split adds the tiles)
    tma_base.maps = plan->tma_maps.empty() ? nullptr : plan->tma_maps.data();
    tma_base.nmaps = static_cast<int32_t>(plan->tma_maps.size());
    tma_base.err = plan->d_err;
    L.tma = plan->tma_maps.empty() ? nullptr : &tma_base;
    // halves: the list for the kinds that run on x-halves (null: none)
    auto launch_list = [&](const DevList &list, const DevList *halves) -> cudaError_t {
        return launch_split(L, list, halves, plan->esize, kinds, stream);
    };
    cudaError_t ce;
    if (mode == COSTA_MODE_DIRECT) {
        ce = mark(0);
        if (ce == cudaSuccess) ce = launch_list(plan->direct, &plan->direct_halves);
        if (ce == cudaSuccess) ce = mark(1);
        if (ce != cudaSuccess) return cuda_fail(ce, "remap kernel launch");
        if (timer) timer->nphases = 1;
        return done(COSTA_OK);
    }
    s = ensure_message(*plan, relabel != 0);
    if (s != COSTA_OK) return s;
    const MessageData &m = plan->msg[relabel ? 1 : 0];
    RemapLaunch lp{};
    lp.tiles = m.pack.tiles;
    lp.ntiles = m.pack.ntiles;
    lp.mtiles = m.pack.mtiles;
    lp.nmtiles = m.pack.nmtiles;
    lp.pieces = m.pack.pieces;
    lp.groups = m.pack.groups;
    lp.ngroups = m.pack.ngroups;
    lp.dtype = plan->dtype;
    lp.per_problem = nullptr;
    const float one_f[2] = {1.0f, 0.0f}, zero_f[2] = {0.0f, 0.0f};
    const double one_d[2] = {1.0, 0.0}, zero_d[2] = {0.0, 0.0};
    const bool single = plan->dtype == COSTA_F32 || plan->dtype == COSTA_C64;
    lp.s = make_scalars(plan->dtype, single ? static_cast<const void *>(one_f) : one_d,
                        single ? static_cast<const void *>(zero_f) : zero_d, 0);
    ce = mark(0);
    if (ce == cudaSuccess) ce = launch_remap(lp, K_COPY, stream);
    if (ce == cudaSuccess) ce = mark(1);
    if (ce != cudaSuccess) return cuda_fail(ce, "pack kernel launch");
    ce = launch_list(m.local, &m.local_halves);
    if (ce == cudaSuccess) ce = mark(2);
    if (ce != cudaSuccess) return cuda_fail(ce, "local remap kernel launch");
    ce = launch_list(m.unpack, &m.unpack_halves);
    if (ce == cudaSuccess) ce = mark(3);
    if (ce != cudaSuccess) return cuda_fail(ce, "unpack kernel launch");
    if (timer) timer->nphases = 3;
    return done(COSTA_OK);
}

costa_status create_layout(costa_layout *out, int dt, int nranks, int nbr, const int64_t *R, int nbc,
                           const int64_t *C, const int *owners, const costa_block *blocks) {
    if (!out) return fail(COSTA_ERR_INVALID_ARG, "out is null");
    *out = nullptr;
    const int es = esize_of(dt);
    if (!es) return fail(COSTA_ERR_DTYPE, "unknown dtype %d", dt);
    if (nranks < 1) return fail(COSTA_ERR_INVALID_ARG, "nranks %d < 1", nranks);
    if (nbr < 0 || nbc < 0) return fail(COSTA_ERR_INVALID_ARG, "negative block counts");
    if (!R || !C) return fail(COSTA_ERR_INVALID_ARG, "null splits");
    const int64_t nblk = static_cast<int64_t>(nbr) * nbc;
    if (nblk > 0 && (!owners || !blocks)) return fail(COSTA_ERR_INVALID_ARG, "null owners or blocks");
    if (R[0] != 0 || C[0] != 0) return fail(COSTA_ERR_LAYOUT, "splits must start at 0");
    for (int i = 0; i < nbr; ++i)
        if (R[i + 1] < R[i]) return fail(COSTA_ERR_LAYOUT, "row splits not sorted at %d", i);
    for (int j = 0; j < nbc; ++j)
        if (C[j + 1] < C[j]) return fail(COSTA_ERR_LAYOUT, "column splits not sorted at %d", j);
    for (int i = 0; i < nbr; ++i)
        if (R[i + 1] - R[i] >= (int64_t(1) << 31)) return fail(COSTA_ERR_LAYOUT, "block row %d too tall", i);
    for (int j = 0; j < nbc; ++j)
        if (C[j + 1] - C[j] >= (int64_t(1) << 31)) return fail(COSTA_ERR_LAYOUT, "block column %d too wide", j);
    auto L = std::make_unique<costa_layout_s>();
    L->id = g_next_id.fetch_add(1);
    L->dt = static_cast<costa_dtype>(dt);
    L->nranks = nranks;
    L->nbr = nbr;
    L->nbc = nbc;
    L->m = R[nbr];
    L->n = C[nbc];
    L->R.assign(R, R + nbr + 1);
    L->C.assign(C, C + nbc + 1);
    L->owner.resize(static_cast<size_t>(nblk));
    L->blocks.resize(static_cast<size_t>(nblk));
    for (int i = 0; i < nbr; ++i) {
        const int64_t h = R[i + 1] - R[i];
        for (int j = 0; j < nbc; ++j) {
            const int64_t w = C[j + 1] - C[j];
            const int64_t b = static_cast<int64_t>(i) * nbc + j;
            if (owners[b] < 0 || owners[b] >= nranks)
                return fail(COSTA_ERR_LAYOUT, "owner %d of block (%d, %d) not in [0, %d)", owners[b], i, j,
                            nranks);
            L->owner[b] = owners[b];
            const costa_block &blk = blocks[b];
            DevBlock d{reinterpret_cast<uint64_t>(blk.ptr), 0, blk.order};
            if (h > 0 && w > 0) {
                if (blk.order != COSTA_COL_MAJOR && blk.order != COSTA_ROW_MAJOR)
                    return fail(COSTA_ERR_LAYOUT, "block (%d, %d): bad order %d", i, j, blk.order);
                if (blk.reserved != 0) return fail(COSTA_ERR_LAYOUT, "block (%d, %d): reserved != 0", i, j);
                // a null pointer: the block's rank keeps its storage in another
                // process (multi-GPU exchange); calls that would read or write
                // the block reject it (check_access, check_blocks_on)
                if (reinterpret_cast<uintptr_t>(blk.ptr) % es)
                    return fail(COSTA_ERR_LAYOUT, "block (%d, %d): pointer not aligned to %d bytes", i, j, es);
                const int64_t need = blk.order == COSTA_COL_MAJOR ? h : w;
                if (blk.ld < need)
                    return fail(COSTA_ERR_LAYOUT, "block (%d, %d): ld %lld < %lld", i, j, (long long)blk.ld,
                                (long long)need);
                if (blk.ld >= (int64_t(1) << 31))
                    return fail(COSTA_ERR_LAYOUT, "block (%d, %d): ld %lld >= 2^31", i, j, (long long)blk.ld);
                d.ld = static_cast<int32_t>(blk.ld);
            } else {
                d.ld = 1;
                d.order = COSTA_COL_MAJOR;
            }
            L->blocks[b] = d;
        }
    }
    *out = L.release();
    return COSTA_OK;
}

int64_t numroc(int64_t n, int64_t nb, int iproc, int nprocs) {
    const int64_t nblocks = n / nb;
    int64_t r = (nblocks / nprocs) * nb;
    const int64_t extra = nblocks % nprocs;
    if (iproc < extra) r += nb;
    else if (iproc == extra) r += n % nb;
    return r;
}

}  // namespace

// Every tile of a list fits the kernel's tile extent along both axes (the
// kernel's shared-memory buffers and register passes are sized by it).
costa_status check_extents(const std::vector<TileDesc> &list, int es, const char *what) {
    const int ts = tile_extent(es);
    for (const TileDesc &d : list)
        if (d.nx < 1 || d.ny < 1 || d.nx > ts || d.ny > ts)
            return fail(COSTA_ERR_INTERNAL, "%s tile %d x %d exceeds the tile extent %d", what, d.nx, d.ny, ts);
    return COSTA_OK;
}

void read_scalar(int dt, const void *p, int index, double out[2]) {
    switch (dt) {
    case COSTA_F32: out[0] = static_cast<const float *>(p)[index]; out[1] = 0.0; break;
    case COSTA_F64: out[0] = static_cast<const double *>(p)[index]; out[1] = 0.0; break;
    case COSTA_C64:
        out[0] = static_cast<const float *>(p)[2 * index];
        out[1] = static_cast<const float *>(p)[2 * index + 1];
        break;
    default:
        out[0] = static_cast<const double *>(p)[2 * index];
        out[1] = static_cast<const double *>(p)[2 * index + 1];
        break;
    }
}

Scalars make_scalars(int dt, const void *alpha, const void *beta, int index) {
    Scalars s{};
    read_scalar(dt, alpha, index, s.alpha);
    read_scalar(dt, beta, index, s.beta);
    s.flags = 0;
    if (s.beta[0] == 0.0 && s.beta[1] == 0.0) s.flags |= SF_BETA0;
    if (s.alpha[0] == 1.0 && s.alpha[1] == 0.0) s.flags |= SF_ALPHA1;
    if (s.alpha[1] != 0.0 || s.beta[1] != 0.0) s.flags |= SF_CPLX;
    int e = 0;
    const double fr = std::frexp(std::fabs(s.beta[0]), &e);
    if (s.beta[1] == 0.0 && fr == 0.5 && e - 1 >= -1000 && e - 1 <= 1000) {
        s.flags |= SF_BPOW2;  // |beta| = 2^(e-1)
        s.beta_exp = e - 1;
    }
    return s;
}

cudaError_t launch_split(const RemapLaunch &base, const DevList &list, const DevList *halves, int esize,
                         const bool (&kinds)[K_NKINDS], cudaStream_t stream) {
    RemapLaunch l = base;
    l.tiles = list.tiles;
    l.ntiles = list.ntiles;
    l.tma = nullptr;
    TmaLists tl{};
    if (base.tma) tl = *base.tma;  // the plan's maps and error word
    l.mtiles = list.mtiles;
    l.nmtiles = list.nmtiles;
    l.pieces = list.pieces;
    l.groups = list.groups;
    l.ngroups = list.ngroups;
    for (int kind = 0; kind < K_NKINDS; ++kind) {
        if (!kinds[kind]) continue;
        RemapLaunch lk = l;
        const DevList &full = (halves && (esize == 4 || kind == K_AXPBY2)) ? *halves : list;
        lk.tiles = full.tiles;
        lk.ntiles = full.ntiles;
        if (base.tma && ((full.tma_kinds >> kind) & 1u)) {  // this kind takes the TMA split
            lk.tiles = full.rtiles;
            lk.ntiles = full.nrtiles;
            tl.ttiles = full.ttiles;
            tl.nttiles = full.nttiles;
            lk.tma = &tl;
        }
        if (kind_reads_a(kind)) {  // the groups of the kinds that read A
            lk.groups = list.groups_a;
            lk.ngroups = list.ngroups_a;
        }
        cudaError_t e = launch_remap(lk, kind, stream);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

costa_status report_error(costa_status s, const char *message) { return fail(s, "%s", message); }

int log_level() {
    static const int level = [] {
        const char *e = std::getenv("COSTA_LOG");
        return e ? std::max(0, std::atoi(e)) : 0;
    }();
    return level;
}

void log_msg(int level, const char *fmt, ...) {
    if (log_level() < level) return;
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    std::fprintf(stderr, "[costa] %s\n", buf);
}

costa_status check_access_on(costa_layout_s *L, int dev, const char *which, const int *place, int g) {
    return check_access_impl(L, dev, which, place, g);
}

costa_status check_pair(const costa_layout_s *A, const costa_layout_s *B, int op) {
    return validate_pair(A, B, op);
}

}  // namespace costa

using namespace costa;

extern "C" {

costa_status costa_layout_create(costa_layout *out, costa_dtype dt, int nranks, int nbr,
                                 const int64_t *row_splits, int nbc, const int64_t *col_splits,
                                 const int *owners, const costa_block *blocks) {
    return create_layout(out, dt, nranks, nbr, row_splits, nbc, col_splits, owners, blocks);
}

costa_status costa_layout_create_block_cyclic(costa_layout *out, costa_dtype dt, int64_t m, int64_t n,
                                              int64_t mb, int64_t nb, int pr, int pc, char grid_order,
                                              const int *rank_perm, void *const *rank_ptrs,
                                              const int64_t *lld) {
    if (!out) return fail(COSTA_ERR_INVALID_ARG, "out is null");
    *out = nullptr;
    if (m < 0 || n < 0 || mb < 1 || nb < 1 || pr < 1 || pc < 1)
        return fail(COSTA_ERR_INVALID_ARG, "bad block-cyclic sizes");
    if (grid_order != 'R' && grid_order != 'C') return fail(COSTA_ERR_INVALID_ARG, "grid_order must be 'R' or 'C'");
    if (!rank_ptrs || !lld) return fail(COSTA_ERR_INVALID_ARG, "null rank pointers or lld");
    const int P = pr * pc;
    const int es = esize_of(dt);
    if (!es) return fail(COSTA_ERR_DTYPE, "unknown dtype %d", dt);
    std::vector<int> perm(P);
    std::vector<char> seen(P, 0);
    for (int r = 0; r < P; ++r) {
        perm[r] = rank_perm ? rank_perm[r] : r;
        if (perm[r] < 0 || perm[r] >= P || seen[perm[r]])
            return fail(COSTA_ERR_LAYOUT, "rank_perm is not a permutation of [0, %d)", P);
        seen[perm[r]] = 1;
    }
    const int64_t nbr64 = (m + mb - 1) / mb, nbc64 = (n + nb - 1) / nb;
    if (nbr64 > (1 << 30) || nbc64 > (1 << 30)) return fail(COSTA_ERR_INVALID_ARG, "too many blocks");
    const int nbr = static_cast<int>(nbr64), nbc = static_cast<int>(nbc64);
    std::vector<int64_t> R(nbr + 1), C(nbc + 1);
    for (int i = 0; i <= nbr; ++i) R[i] = std::min<int64_t>(i * mb, m);
    for (int j = 0; j <= nbc; ++j) C[j] = std::min<int64_t>(j * nb, n);
    std::vector<int> owners(static_cast<size_t>(nbr) * nbc);
    std::vector<costa_block> blocks(static_cast<size_t>(nbr) * nbc);
    for (int bi = 0; bi < nbr; ++bi) {
        const int i = bi % pr;
        for (int bj = 0; bj < nbc; ++bj) {
            const int j = bj % pc;
            const int grank = grid_order == 'R' ? i * pc + j : i + j * pr;
            const int o = perm[grank];
            const size_t b = static_cast<size_t>(bi) * nbc + bj;
            owners[b] = o;
            const int64_t lr = static_cast<int64_t>(bi / pr) * mb, lc = static_cast<int64_t>(bj / pc) * nb;
            const int64_t need = numroc(m, mb, i, pr);
            if (lld[o] < std::max<int64_t>(1, need))
                return fail(COSTA_ERR_LAYOUT, "lld[%d] = %lld < local rows %lld", o, (long long)lld[o],
                            (long long)need);
            // a null rank pointer: that rank's storage lives in another process
            blocks[b].ptr = rank_ptrs[o] ? static_cast<char *>(rank_ptrs[o]) + (lr + lc * lld[o]) * es : nullptr;
            blocks[b].ld = lld[o];
            blocks[b].order = COSTA_COL_MAJOR;
            blocks[b].reserved = 0;
        }
    }
    return create_layout(out, dt, P, nbr, R.data(), nbc, C.data(), owners.data(), blocks.data());
}

costa_status costa_layout_destroy(costa_layout layout) {
    if (!layout) return COSTA_OK;
    {
        std::lock_guard<std::mutex> lock(g_mu);
        for (auto it = g_plans.begin(); it != g_plans.end();) {
            if (plan_uses(it->first, layout->id)) it = g_plans.erase(it);
            else ++it;
        }
    }
    delete layout;
    return COSTA_OK;
}

costa_status costa_layout_info(costa_layout layout, int64_t *m, int64_t *n, int *nranks, int *dtype) {
    if (!layout) return fail(COSTA_ERR_INVALID_ARG, "null layout");
    if (m) *m = layout->m;
    if (n) *n = layout->n;
    if (nranks) *nranks = layout->nranks;
    if (dtype) *dtype = layout->dt;
    return COSTA_OK;
}

costa_status costa_volume(costa_layout A, costa_layout B, costa_op op, int64_t *V, void *stream) {
    costa_status s = validate_pair(A, B, op);
    if (s != COSTA_OK) return s;
    if (!V) return fail(COSTA_ERR_INVALID_ARG, "V is null");
    std::lock_guard<std::mutex> lock(g_mu);
    Plan *plan = nullptr;
    s = get_plan(1, &A, &B, &op, static_cast<cudaStream_t>(stream), plan);
    if (s != COSTA_OK) return s;
    std::memcpy(V, plan->V.data(), sizeof(int64_t) * plan->V.size());
    return COSTA_OK;
}

costa_status costa_relabel(int P, const int64_t *V, int *sigma, int64_t *local_volume) {
    if (P < 1) return fail(COSTA_ERR_INVALID_ARG, "P %d < 1", P);
    if (!V || !sigma) return fail(COSTA_ERR_INVALID_ARG, "null argument");
    for (int64_t k = 0; k < static_cast<int64_t>(P) * P; ++k)
        if (V[k] < 0) return fail(COSTA_ERR_INVALID_ARG, "negative volume at %lld", (long long)k);
    std::vector<int> sig;
    int64_t best = 0;
    solve_relabel(P, V, sig, best);
    std::copy(sig.begin(), sig.end(), sigma);
    if (local_volume) *local_volume = best;
    return COSTA_OK;
}

// Relabeling under the topology cost of Sec. 3: w(i, j, s) = lat[i][j] +
// bw[i][j] * V(s) for i != j, 0 for i == j, and nothing for empty packages.
// As in Alg. 1 the weights are the gains of Eq. 3,
//   delta(x, y) = sum over senders i of package S_ix of w(i, x, S_ix) - w(i, y, S_ix),
// and sigma maximizes sum_x delta(x, sigma(x)) (Thm. 1), solved exactly as an
// assignment on doubles.  By Lemma 1 this minimizes W(G_sigma).
costa_status costa_relabel_cost(int P, const int64_t *V, const double *lat, const double *bw, int *sigma,
                                double *cost_identity, double *cost_relabeled) {
    if (P < 1) return fail(COSTA_ERR_INVALID_ARG, "P %d < 1", P);
    if (!V || !lat || !bw || !sigma) return fail(COSTA_ERR_INVALID_ARG, "null argument");
    const size_t PP = static_cast<size_t>(P) * P;
    for (size_t k = 0; k < PP; ++k) {
        if (V[k] < 0) return fail(COSTA_ERR_INVALID_ARG, "negative volume at %zu", k);
        if (!std::isfinite(lat[k]) || !std::isfinite(bw[k]))
            return fail(COSTA_ERR_INVALID_ARG, "non-finite cost at %zu", k);
    }
    auto w = [&](int i, int j, int64_t v) -> double {
        if (v == 0 || i == j) return 0.0;
        return lat[static_cast<size_t>(i) * P + j] + bw[static_cast<size_t>(i) * P + j] * static_cast<double>(v);
    };
    // C[x][y]: cost of the packages of target label x when process y takes it
    std::vector<double> C(PP, 0.0);
    for (int x = 0; x < P; ++x)
        for (int y = 0; y < P; ++y) {
            double c = 0.0;
            for (int i = 0; i < P; ++i) c += w(i, y, V[static_cast<size_t>(i) * P + x]);
            C[static_cast<size_t>(x) * P + y] = c;
        }
    // maximize sum delta(x, sigma(x)) with delta(x, y) = C[x][x] - C[x][y]:
    // the same assignment as minimizing sum C[x][sigma(x)]
    std::vector<double> cost(PP);
    for (int x = 0; x < P; ++x)
        for (int y = 0; y < P; ++y)
            cost[static_cast<size_t>(x) * P + y] =
                -(C[static_cast<size_t>(x) * P + x] - C[static_cast<size_t>(x) * P + y]);
    std::vector<int> row_to_col;
    assign_min_f(P, cost, row_to_col);
    double ident = 0.0, best = 0.0;
    for (int x = 0; x < P; ++x) {
        ident += C[static_cast<size_t>(x) * P + x];
        best += C[static_cast<size_t>(x) * P + row_to_col[x]];
    }
    const bool keep = ident <= best;  // tie rule: the identity when it is optimal
    for (int x = 0; x < P; ++x) sigma[x] = keep ? x : row_to_col[x];
    if (cost_identity) *cost_identity = ident;
    if (cost_relabeled) *cost_relabeled = keep ? ident : best;
    return COSTA_OK;
}

costa_status costa_relabel_placement(int P, const int64_t *V, int G, const int *place, double intra, int *sigma,
                                     double *cost_identity, double *cost_relabeled) {
    if (P < 1) return fail(COSTA_ERR_INVALID_ARG, "P %d < 1", P);
    if (G < 1 || !place) return fail(COSTA_ERR_INVALID_ARG, "G < 1 or null placement");
    if (!std::isfinite(intra) || intra < 0.0) return fail(COSTA_ERR_INVALID_ARG, "intra must be finite and >= 0");
    for (int r = 0; r < P; ++r)
        if (place[r] < 0 || place[r] >= G) return fail(COSTA_ERR_INVALID_ARG, "place[%d] not in [0, %d)", r, G);
    const size_t PP = static_cast<size_t>(P) * P;
    std::vector<double> lat(PP, 0.0), bw(PP, 0.0);
    for (int i = 0; i < P; ++i)
        for (int k = 0; k < P; ++k)
            if (i != k) bw[static_cast<size_t>(i) * P + k] = place[i] == place[k] ? intra : 1.0;
    return costa_relabel_cost(P, V, lat.data(), bw.data(), sigma, cost_identity, cost_relabeled);
}

costa_status costa_relabel_greedy(int P, const int64_t *V, int *sigma, int64_t *local_volume) {
    if (P < 1) return fail(COSTA_ERR_INVALID_ARG, "P %d < 1", P);
    if (!V || !sigma) return fail(COSTA_ERR_INVALID_ARG, "null argument");
    for (int64_t k = 0; k < static_cast<int64_t>(P) * P; ++k)
        if (V[k] < 0) return fail(COSTA_ERR_INVALID_ARG, "negative volume at %lld", (long long)k);
    std::vector<int> sig;
    const int64_t total = greedy_max(P, V, sig);
    std::copy(sig.begin(), sig.end(), sigma);
    if (local_volume) *local_volume = total;
    return COSTA_OK;
}

costa_status costa_transform(costa_layout A, costa_layout B, costa_op op, const void *alpha, const void *beta,
                             int relabel, int *sigma_out, void *stream) {
    return transform_impl(1, &A, &B, &op, alpha, beta, relabel, sigma_out, COSTA_MODE_DIRECT, stream);
}

costa_status costa_transform_ex(costa_layout A, costa_layout B, costa_op op, const void *alpha,
                                const void *beta, int relabel, int *sigma_out, costa_mode mode,
                                void *stream) {
    return transform_impl(1, &A, &B, &op, alpha, beta, relabel, sigma_out, mode, stream);
}

costa_status costa_transform_batched(int n, const costa_layout *A, const costa_layout *B, const costa_op *ops,
                                     const void *alphas, const void *betas, int relabel, int *sigma_out,
                                     void *stream) {
    return transform_impl(n, A, B, ops, alphas, betas, relabel, sigma_out, COSTA_MODE_DIRECT, stream);
}

costa_status costa_transform_batched_ex(int n, const costa_layout *A, const costa_layout *B,
                                        const costa_op *ops, const void *alphas, const void *betas,
                                        int relabel, int *sigma_out, costa_mode mode, void *stream) {
    return transform_impl(n, A, B, ops, alphas, betas, relabel, sigma_out, mode, stream);
}

costa_status costa_plan_stats_get(int n, const costa_layout *A, const costa_layout *B, const costa_op *ops,
                                  int relabel, costa_plan_stats *stats, void *stream) {
    if (n < 1 || !A || !B || !ops || !stats) return fail(COSTA_ERR_INVALID_ARG, "bad arguments");
    for (int k = 0; k < n; ++k) {
        costa_status s = validate_pair(A[k], B[k], ops[k]);
        if (s != COSTA_OK) return s;
    }
    std::lock_guard<std::mutex> lock(g_mu);
    Plan *plan = nullptr;
    costa_status s = get_plan(n, A, B, ops, static_cast<cudaStream_t>(stream), plan);
    if (s != COSTA_OK) return s;
    if (relabel) {
        s = ensure_sigma(*plan);
        if (s != COSTA_OK) return s;
    }
    *stats = plan->stats;
    if (!relabel) stats->local_relabeled = stats->local_identity;
    stats->staging_bytes = plan->msg[relabel ? 1 : 0].built ? plan->msg[relabel ? 1 : 0].staging_bytes : -1;
    return COSTA_OK;
}

costa_status costa_debug_axis_pieces(costa_layout A, costa_layout B, costa_op op, int axis, int32_t *out,
                                     int64_t cap, int64_t *count) {
    costa_status s = validate_pair(A, B, op);
    if (s != COSTA_OK) return s;
    if ((axis != 0 && axis != 1) || !count || (cap > 0 && !out))
        return fail(COSTA_ERR_INVALID_ARG, "bad arguments");
    const AxisCut cut = cut_pair_axis(A, B, op, axis, tile_extent(esize_of(A->dt)));
    *count = static_cast<int64_t>(cut.tiles.size());
    for (int64_t k = 0; k < std::min<int64_t>(cap, *count); ++k) {
        const AxisTile &t = cut.tiles[static_cast<size_t>(k)];
        const int32_t v[6] = {t.a_blk, t.b_blk, t.a_off, t.b_off, t.len, t.cell};
        std::memcpy(out + 6 * k, v, sizeof v);
    }
    return COSTA_OK;
}

costa_status costa_debug_tiles(costa_layout A, costa_layout B, costa_op op, void *out, int64_t cap,
                               int64_t *count) {
    costa_status s = validate_pair(A, B, op);
    if (s != COSTA_OK) return s;
    if (!count || (cap > 0 && !out)) return fail(COSTA_ERR_INVALID_ARG, "bad arguments");
    const int es = esize_of(A->dt), ts = tile_extent(es);
    ProblemHost ph;
    ph.A = A;
    ph.B = B;
    ph.op = op;
    ph.rows = cut_pair_axis(A, B, op, 0, ts);
    ph.cols = cut_pair_axis(A, B, op, 1, ts);
    *count = static_cast<int64_t>(ph.rows.tiles.size()) * static_cast<int64_t>(ph.cols.tiles.size());
    std::vector<TileDesc> list;
    list.reserve(static_cast<size_t>(*count));
    append_direct_tiles(ph, 0, es, ts, list);
    const size_t k = static_cast<size_t>(std::min<int64_t>(cap, *count));
    if (k) std::memcpy(out, list.data(), k * sizeof(TileDesc));
    return COSTA_OK;
}

costa_status costa_debug_split(costa_layout A, costa_layout B, costa_op op, void *tiles, int64_t cap_tiles,
                               void *pieces, int64_t cap_pieces, uint32_t *groups, int64_t cap_groups,
                               int64_t *ntiles, int64_t *npieces, int64_t *ngroups) {
    costa_status s = validate_pair(A, B, op);
    if (s != COSTA_OK) return s;
    if (!ntiles || !npieces || !ngroups || (cap_tiles > 0 && !tiles) || (cap_pieces > 0 && !pieces) ||
        (cap_groups > 0 && !groups))
        return fail(COSTA_ERR_INVALID_ARG, "bad arguments");
    const int es = esize_of(A->dt), ts = tile_extent(es);
    ProblemHost ph;
    ph.A = A;
    ph.B = B;
    ph.op = op;
    ph.rows = cut_pair_axis(A, B, op, 0, ts);
    ph.cols = cut_pair_axis(A, B, op, 1, ts);
    std::vector<TileDesc> list;
    append_direct_tiles(ph, 0, es, ts, list);
    const SplitList sp = split_small(std::move(list), es, A->dt == COSTA_C64 || A->dt == COSTA_C128);
    std::vector<TileDesc> whole = sp.big;  // the tile kernel's tiles: aligned, then misaligned
    whole.insert(whole.end(), sp.mis.begin(), sp.mis.end());
    *ntiles = static_cast<int64_t>(whole.size());
    *npieces = static_cast<int64_t>(sp.pieces.size());
    *ngroups = sp.ngroups();
    const size_t kt = static_cast<size_t>(std::min<int64_t>(cap_tiles, *ntiles));
    const size_t kp = static_cast<size_t>(std::min<int64_t>(cap_pieces, *npieces));
    const size_t kg = static_cast<size_t>(std::min<int64_t>(cap_groups, static_cast<int64_t>(sp.groups.size())));
    if (kt) std::memcpy(tiles, whole.data(), kt * sizeof(TileDesc));
    if (kp) std::memcpy(pieces, sp.pieces.data(), kp * sizeof(TileDesc));
    if (kg) std::memcpy(groups, sp.groups.data(), kg * sizeof(uint32_t));
    return COSTA_OK;
}

costa_status costa_debug_groups(costa_layout A, costa_layout B, costa_op op, int reads_a, uint32_t *groups,
                                int64_t cap_groups, int64_t *ngroups) {
    costa_status s = validate_pair(A, B, op);
    if (s != COSTA_OK) return s;
    if (!ngroups || (cap_groups > 0 && !groups)) return fail(COSTA_ERR_INVALID_ARG, "bad arguments");
    const int es = esize_of(A->dt), ts = tile_extent(es);
    ProblemHost ph;
    ph.A = A;
    ph.B = B;
    ph.op = op;
    ph.rows = cut_pair_axis(A, B, op, 0, ts);
    ph.cols = cut_pair_axis(A, B, op, 1, ts);
    std::vector<TileDesc> list;
    append_direct_tiles(ph, 0, es, ts, list);
    const SplitList sp = split_small(std::move(list), es, A->dt == COSTA_C64 || A->dt == COSTA_C128);
    const std::vector<uint32_t> &g = reads_a ? sp.groups_a : sp.groups;
    *ngroups = reads_a ? sp.ngroups_a() : sp.ngroups();
    const size_t k = static_cast<size_t>(std::min<int64_t>(cap_groups, static_cast<int64_t>(g.size())));
    if (k) std::memcpy(groups, g.data(), k * sizeof(uint32_t));
    return COSTA_OK;
}

costa_status costa_debug_halves(costa_layout A, costa_layout B, costa_op op, void *tiles, int64_t cap_tiles,
                                int64_t *ntiles) {
    costa_status s = validate_pair(A, B, op);
    if (s != COSTA_OK) return s;
    if (!ntiles || (cap_tiles > 0 && !tiles)) return fail(COSTA_ERR_INVALID_ARG, "bad arguments");
    const int es = esize_of(A->dt), ts = tile_extent(es);
    ProblemHost ph;
    ph.A = A;
    ph.B = B;
    ph.op = op;
    ph.rows = cut_pair_axis(A, B, op, 0, ts);
    ph.cols = cut_pair_axis(A, B, op, 1, ts);
    std::vector<TileDesc> list;
    append_direct_tiles(ph, 0, es, ts, list);
    const SplitList sp = split_small(std::move(list), es, A->dt == COSTA_C64 || A->dt == COSTA_C128);
    const std::vector<TileDesc> halves =
        split_x_halves(sp.big, ts / 2, es, std::vector<char>(1, use_halves(ph, es) ? 1 : 0));
    *ntiles = static_cast<int64_t>(halves.size());
    const size_t k = static_cast<size_t>(std::min<int64_t>(cap_tiles, *ntiles));
    if (k) std::memcpy(tiles, halves.data(), k * sizeof(TileDesc));
    return COSTA_OK;
}

costa_status costa_debug_tma(costa_layout A, costa_layout B, costa_op op, int64_t *out) {
    if (!out) return fail(COSTA_ERR_INVALID_ARG, "out is null");
    costa_status s = validate_pair(A, B, op);
    if (s != COSTA_OK) return s;
    std::lock_guard<std::mutex> lock(g_mu);
    Plan *plan = nullptr;
    s = get_plan(1, &A, &B, &op, nullptr, plan);
    if (s == COSTA_OK) s = ensure_tma(*plan);
    if (s != COSTA_OK) return s;
    unsigned int err = 0;
    cudaError_t ce = cudaMemcpy(&err, plan->d_err, sizeof err, cudaMemcpyDeviceToHost);
    if (ce != cudaSuccess) return cuda_fail(ce, "cudaMemcpy(error word)");
    out[0] = plan->direct.nttiles;
    out[1] = plan->direct_halves.ttiles == plan->direct.ttiles ? 0 : plan->direct_halves.nttiles;
    out[4] = plan->direct.tma_kinds;
    out[5] = plan->direct_halves.ttiles == plan->direct.ttiles ? 0 : plan->direct_halves.tma_kinds;
    out[2] = static_cast<int64_t>(plan->tma_maps.size());
    out[3] = err;
    return COSTA_OK;
}

costa_status costa_debug_fxdot(int n, int64_t count, const double *x, const double *y, const int32_t *neg,
                               double *out) {
    if ((n != 2 && n != 4) || count < 0 || (count > 0 && (!x || !y || !neg || !out)))
        return fail(COSTA_ERR_INVALID_ARG, "costa_debug_fxdot: n must be 2 or 4 and the arrays non-null");
    for (int64_t k = 0; k < count * n; ++k)
        if (!fx::in_range(x[k]) || !fx::in_range(y[k]))
            return fail(COSTA_ERR_INVALID_ARG, "costa_debug_fxdot: factor %lld is outside [2^-480, 2^480)",
                        (long long)k);
    for (int64_t k = 0; k < count; ++k) {
        const double *xk = x + k * n, *yk = y + k * n;
        const int32_t *nk = neg + k * n;
        if (n == 2) {
            const fx::Term t[2] = {fx::mul(fx::unpack(xk[0]), fx::unpack(yk[0]), nk[0] ? 1u : 0u),
                                   fx::mul(fx::unpack(xk[1]), fx::unpack(yk[1]), nk[1] ? 1u : 0u)};
            out[k] = fx::sum(t);
        } else {
            fx::Term t[4];
            for (int i = 0; i < 4; ++i) t[i] = fx::mul(fx::unpack(xk[i]), fx::unpack(yk[i]), nk[i] ? 1u : 0u);
            out[k] = fx::sum(t);
        }
    }
    return COSTA_OK;
}

costa_status costa_release_plans(void) {
    std::lock_guard<std::mutex> lock(g_mu);
    g_plans.clear();
    return COSTA_OK;
}

const char *costa_last_error(void) { return g_err.c_str(); }

int64_t costa_kernel_launch_count(void) { return launches_so_far(); }

costa_status costa_phase_timing(int enable) {
    g_phase_on.store(enable != 0);
    return COSTA_OK;
}

costa_status costa_phase_times(double *ms, int *nphases) {
    if (!ms || !nphases) return fail(COSTA_ERR_INVALID_ARG, "null argument");
    std::lock_guard<std::mutex> lock(g_mu);
    costa_status st;
    PhaseTimer *t = phase_timer(st);
    if (!t) return st;
    if (t->nphases == 0) return fail(COSTA_ERR_INVALID_ARG, "no timed transform call with tiles on this device");
    cudaError_t ce = cudaEventSynchronize(t->ev[t->nphases]);
    if (ce != cudaSuccess) return cuda_fail(ce, "cudaEventSynchronize");
    for (int k = 0; k < t->nphases; ++k) {
        float f = 0.0f;
        ce = cudaEventElapsedTime(&f, t->ev[k], t->ev[k + 1]);
        if (ce != cudaSuccess) return cuda_fail(ce, "cudaEventElapsedTime");
        ms[k] = f;
    }
    *nphases = t->nphases;
    return COSTA_OK;
}

int costa_abi_version(void) { return 1; }

}  // extern "C"
