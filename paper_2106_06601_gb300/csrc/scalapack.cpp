// ScaLAPACK-style entry points (Sec. 6: "provides the ScaLAPACK wrappers for
// pxgemr2d and pxtran"): submatrices of 2D block-cyclic matrices given by
// ScaLAPACK array descriptors, on a grid of virtual ranks.
//
// A submatrix is a layout of its own: the global block grid truncated to the
// submatrix's rows and columns (Sec. 5: "first truncate the corresponding
// row-splits and column-splits"), each block pointing into its owner's local
// matrix at the ScaLAPACK local indices.  The transforms then run through
// costa_transform on a cache of such layout pairs, so repeated calls with the
// same arguments reuse their plan.
#include <algorithm>
#include <cstdio>
#include <cstring>
#include <list>
#include <mutex>
#include <vector>

#include "costa_gb300.h"
#include "costa_internal.h"

namespace costa {
namespace {

int esize_sl(int dt) { return dt == COSTA_F32 ? 4 : dt == COSTA_C128 ? 16 : dt <= COSTA_C128 ? 8 : 0; }

// Rows of an n-long dimension held by process iproc (NUMROC).
int64_t numroc(int64_t n, int64_t nb, int iproc, int isrc, int nprocs) {
    const int mydist = (nprocs + iproc - isrc) % nprocs;
    const int64_t nblocks = n / nb;
    int64_t r = (nblocks / nprocs) * nb;
    const int64_t extra = nblocks % nprocs;
    if (mydist < extra) r += nb;
    else if (mydist == extra) r += n % nb;
    return r;
}

costa_status bad(costa_status s, const char *msg) { return report_error(s, msg); }

struct PairKey {
    std::vector<int64_t> v;
    bool operator==(const PairKey &o) const { return v == o.v; }
};
struct PairEntry {
    PairKey key;
    costa_layout target = nullptr, source = nullptr;
};
std::mutex g_sl_mu;
std::list<PairEntry> g_sl_cache;  // most recently used first
constexpr size_t kCacheMax = 32;

void key_grid(std::vector<int64_t> &k, const costa_blacs_grid *g) {
    const int P = g->nprow * g->npcol;
    k.push_back(g->nprow);
    k.push_back(g->npcol);
    k.push_back(g->order);
    for (int r = 0; r < P; ++r) {
        k.push_back(static_cast<int64_t>(reinterpret_cast<uintptr_t>(g->local[r])));
        k.push_back(g->lld ? g->lld[r] : -1);
    }
}

}  // namespace
}  // namespace costa

using namespace costa;

extern "C" costa_status costa_layout_create_scalapack(costa_layout *out, costa_dtype dt,
                                                      const costa_blacs_grid *g, int64_t i, int64_t j,
                                                      int64_t m, int64_t n, const int64_t *desc) {
    if (!out) return bad(COSTA_ERR_INVALID_ARG, "out is null");
    *out = nullptr;
    const int es = esize_sl(dt);
    if (!es) return bad(COSTA_ERR_DTYPE, "unknown dtype");
    if (!g || !desc || !g->local || g->nprow < 1 || g->npcol < 1 || (g->order != 'R' && g->order != 'C'))
        return bad(COSTA_ERR_INVALID_ARG, "bad grid or descriptor");
    if (desc[0] != 1) return bad(COSTA_ERR_INVALID_ARG, "descriptor type (DTYPE_) must be 1");
    const int64_t M = desc[2], N = desc[3], MB = desc[4], NB = desc[5];
    const int64_t RSRC = desc[6], CSRC = desc[7], LLD = desc[8];
    const int pr = g->nprow, pc = g->npcol, P = pr * pc;
    if (M < 0 || N < 0 || MB < 1 || NB < 1 || RSRC < 0 || RSRC >= pr || CSRC < 0 || CSRC >= pc)
        return bad(COSTA_ERR_INVALID_ARG, "bad descriptor entries (M, N, MB, NB, RSRC, CSRC)");
    if (m < 0 || n < 0 || i < 1 || j < 1 || i - 1 + m > M || j - 1 + n > N)
        return bad(COSTA_ERR_SHAPE, "submatrix (i, j, m, n) outside the global matrix");
    const int64_t i0 = i - 1, j0 = j - 1;
    // truncated splits: block boundaries of the global grid inside the submatrix
    std::vector<int64_t> R{0}, C{0}, gbr, gbc;  // gbr/gbc: global block index of each sub-block
    for (int64_t r = 0; r < m;) {
        const int64_t gr = i0 + r, gb = gr / MB, end = std::min((gb + 1) * MB - i0, m);
        gbr.push_back(gb);
        R.push_back(end);
        r = end;
    }
    for (int64_t c = 0; c < n;) {
        const int64_t gc = j0 + c, gb = gc / NB, end = std::min((gb + 1) * NB - j0, n);
        gbc.push_back(gb);
        C.push_back(end);
        c = end;
    }
    const int nbr = static_cast<int>(gbr.size()), nbc = static_cast<int>(gbc.size());
    std::vector<int> owners(static_cast<size_t>(nbr) * nbc);
    std::vector<costa_block> blocks(static_cast<size_t>(nbr) * nbc);
    for (int bi = 0; bi < nbr; ++bi) {
        const int prow = static_cast<int>((gbr[bi] + RSRC) % pr);
        const int64_t gr = i0 + R[bi];                                   // first global row
        const int64_t lr = MB * (gr / (MB * pr)) + gr % MB;               // INDXG2L
        for (int bj = 0; bj < nbc; ++bj) {
            const int pcol = static_cast<int>((gbc[bj] + CSRC) % pc);
            const int64_t gc = j0 + C[bj];
            const int64_t lc = NB * (gc / (NB * pc)) + gc % NB;
            const int rank = g->order == 'R' ? prow * pc + pcol : prow + pcol * pr;
            const int64_t lld = g->lld ? g->lld[rank] : LLD;
            const int64_t need = std::max<int64_t>(1, numroc(M, MB, prow, static_cast<int>(RSRC), pr));
            if (lld < need) {
                char msg[160];
                snprintf(msg, sizeof msg, "rank %d: LLD %lld < local rows %lld", rank, (long long)lld,
                         (long long)need);
                return bad(COSTA_ERR_LAYOUT, msg);
            }
            if (!g->local[rank]) return bad(COSTA_ERR_LAYOUT, "null local matrix pointer");
            const size_t b = static_cast<size_t>(bi) * nbc + bj;
            owners[b] = rank;
            blocks[b].ptr = static_cast<char *>(g->local[rank]) + (lr + lc * lld) * es;
            blocks[b].ld = lld;
            blocks[b].order = COSTA_COL_MAJOR;
            blocks[b].reserved = 0;
        }
    }
    (void)P;
    return costa_layout_create(out, dt, pr * pc, nbr, R.data(), nbc, C.data(), owners.data(), blocks.data());
}

namespace {

// The (target, source) layout pair for the given arguments, from the cache.
costa_status get_pair(costa_dtype dt, const costa_blacs_grid *gs, int64_t is, int64_t js, int64_t ms,
                      int64_t ns, const int64_t *ds, const costa_blacs_grid *gt, int64_t it, int64_t jt,
                      int64_t mt, int64_t nt, const int64_t *dt_, costa_layout *target,
                      costa_layout *source) {
    if (!gs || !gt || !ds || !dt_ || !gs->local || !gt->local)
        return bad(COSTA_ERR_INVALID_ARG, "null grid or descriptor");
    PairKey key;
    key.v = {dt, is, js, ms, ns, it, jt, mt, nt};
    for (int k = 0; k < 9; ++k) key.v.push_back(ds[k]);
    for (int k = 0; k < 9; ++k) key.v.push_back(dt_[k]);
    if (gs->nprow < 1 || gs->npcol < 1 || gt->nprow < 1 || gt->npcol < 1)
        return bad(COSTA_ERR_INVALID_ARG, "bad process grid");
    key_grid(key.v, gs);
    key_grid(key.v, gt);
    std::lock_guard<std::mutex> lock(g_sl_mu);
    for (auto it2 = g_sl_cache.begin(); it2 != g_sl_cache.end(); ++it2) {
        if (it2->key == key) {
            g_sl_cache.splice(g_sl_cache.begin(), g_sl_cache, it2);
            *target = g_sl_cache.front().target;
            *source = g_sl_cache.front().source;
            return COSTA_OK;
        }
    }
    PairEntry e;
    e.key = key;
    costa_status s = costa_layout_create_scalapack(&e.source, dt, gs, is, js, ms, ns, ds);
    if (s != COSTA_OK) return s;
    s = costa_layout_create_scalapack(&e.target, dt, gt, it, jt, mt, nt, dt_);
    if (s != COSTA_OK) {
        costa_layout_destroy(e.source);
        return s;
    }
    g_sl_cache.push_front(e);
    while (g_sl_cache.size() > kCacheMax) {  // evict (destroying a layout frees its plans)
        costa_layout_destroy(g_sl_cache.back().target);
        costa_layout_destroy(g_sl_cache.back().source);
        g_sl_cache.pop_back();
    }
    *target = e.target;
    *source = e.source;
    return COSTA_OK;
}

}  // namespace

extern "C" costa_status costa_pxgemr2d(costa_dtype dt, int64_t m, int64_t n, const costa_blacs_grid *ga,
                                       int64_t ia, int64_t ja, const int64_t *desca,
                                       const costa_blacs_grid *gb, int64_t ib, int64_t jb,
                                       const int64_t *descb, void *stream) {
    costa_layout tgt, src;
    costa_status s = get_pair(dt, ga, ia, ja, m, n, desca, gb, ib, jb, m, n, descb, &tgt, &src);
    if (s != COSTA_OK) return s;
    const double one[2] = {1.0, 0.0}, zero[2] = {0.0, 0.0};
    const float onef[2] = {1.0f, 0.0f}, zerof[2] = {0.0f, 0.0f};
    const bool single = dt == COSTA_F32 || dt == COSTA_C64;
    return costa_transform(tgt, src, COSTA_OP_N, single ? static_cast<const void *>(onef) : one,
                           single ? static_cast<const void *>(zerof) : zero, 0, nullptr, stream);
}

extern "C" costa_status costa_pxtran(costa_dtype dt, int conjugate, int64_t m, int64_t n, const void *alpha,
                                     const costa_blacs_grid *ga, int64_t ia, int64_t ja,
                                     const int64_t *desca, const void *beta, const costa_blacs_grid *gc,
                                     int64_t ic, int64_t jc, const int64_t *descc, void *stream) {
    costa_layout tgt, src;
    // sub(C) is m x n, sub(A) is n x m
    costa_status s = get_pair(dt, ga, ia, ja, n, m, desca, gc, ic, jc, m, n, descc, &tgt, &src);
    if (s != COSTA_OK) return s;
    return costa_transform(tgt, src, conjugate ? COSTA_OP_C : COSTA_OP_T, alpha, beta, 0, nullptr, stream);
}

extern "C" costa_status costa_scalapack_release(void) {
    std::lock_guard<std::mutex> lock(g_sl_mu);
    for (auto &e : g_sl_cache) {
        costa_layout_destroy(e.target);
        costa_layout_destroy(e.source);
    }
    g_sl_cache.clear();
    return COSTA_OK;
}
