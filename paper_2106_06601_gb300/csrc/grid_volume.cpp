// Volumes of the reshuffle for grid-product layouts, without enumerating
// overlay cells.
//
// For a layout whose owner map is a product, owner(bi, bj) =
// grid[rowproc(bi)][colproc(bj)] (block-cyclic layouts and any other
// process-grid layout), the package sizes of Alg. 2 factor: every overlay
// cell is an overlay row interval times an overlay column interval, so
//   V[gB(r, c)][gA(r', c')] = Rows[r][r'] * Cols[c][c'],
// where Rows[r][r'] counts the rows whose source process row is r and target
// process row is r' (one merge of the two row-split lists) and Cols likewise.
// The cost is O(block rows + block columns + P^2), independent of the number
// of overlay cells (10^10 for the 10^5 x 10^5 study of Sec. 7.2 with 1 x 1
// source blocks).
#include <algorithm>
#include <cstdio>
#include <cstring>
#include <vector>

#include "costa_gb300.h"
#include "costa_internal.h"

namespace costa {
namespace {

costa_status check_grid(const costa_grid_desc *g, const char *name) {
    char msg[160];
    if (!g) {
        snprintf(msg, sizeof msg, "%s is null", name);
        return report_error(COSTA_ERR_INVALID_ARG, msg);
    }
    if (g->nbr < 0 || g->nbc < 0 || g->pr < 1 || g->pc < 1 || !g->row_splits || !g->col_splits ||
        !g->grid || (g->nbr > 0 && !g->row_procs) || (g->nbc > 0 && !g->col_procs)) {
        snprintf(msg, sizeof msg, "%s: bad sizes or null arrays", name);
        return report_error(COSTA_ERR_INVALID_ARG, msg);
    }
    if (g->row_splits[0] != 0 || g->col_splits[0] != 0) {
        snprintf(msg, sizeof msg, "%s: splits must start at 0", name);
        return report_error(COSTA_ERR_LAYOUT, msg);
    }
    for (int i = 0; i < g->nbr; ++i)
        if (g->row_splits[i + 1] < g->row_splits[i] || g->row_procs[i] < 0 || g->row_procs[i] >= g->pr) {
            snprintf(msg, sizeof msg, "%s: row split or process row %d out of order or range", name, i);
            return report_error(COSTA_ERR_LAYOUT, msg);
        }
    for (int j = 0; j < g->nbc; ++j)
        if (g->col_splits[j + 1] < g->col_splits[j] || g->col_procs[j] < 0 || g->col_procs[j] >= g->pc) {
            snprintf(msg, sizeof msg, "%s: column split or process column %d out of order or range", name, j);
            return report_error(COSTA_ERR_LAYOUT, msg);
        }
    return COSTA_OK;
}

// Rows counted per (source process index, target process index) along one
// axis: SA/PA are the target's splits and process indices (nA blocks), SB/PB
// the source's (nB blocks); out is nprocB x nprocA.
void axis_overlap(const int64_t *SA, const int *PA, int nA, int nprocA, const int64_t *SB, const int *PB,
                  int nB, int64_t extent, std::vector<int64_t> &out) {
    int ka = 0, kb = 0;
    int64_t pos = 0;
    while (pos < extent) {
        while (ka + 1 < nA && SA[ka + 1] <= pos) ++ka;
        while (kb + 1 < nB && SB[kb + 1] <= pos) ++kb;
        const int64_t end = std::min(SA[ka + 1], SB[kb + 1]);
        out[static_cast<size_t>(PB[kb]) * nprocA + PA[ka]] += end - pos;
        pos = end;
    }
}

}  // namespace
}  // namespace costa

using namespace costa;

extern "C" costa_status costa_volume_grid(const costa_grid_desc *A, const costa_grid_desc *B, costa_op op,
                                          int P, int64_t *V) {
    costa_status s = check_grid(A, "A");
    if (s != COSTA_OK) return s;
    s = check_grid(B, "B");
    if (s != COSTA_OK) return s;
    if (op < COSTA_OP_N || op > COSTA_OP_C) return report_error(COSTA_ERR_INVALID_ARG, "bad op");
    if (!V || P < 1) return report_error(COSTA_ERR_INVALID_ARG, "V is null or P < 1");
    const bool tr = op != COSTA_OP_N;
    const int64_t mA = A->row_splits[A->nbr], nA = A->col_splits[A->nbc];
    const int64_t mB = B->row_splits[B->nbr], nB = B->col_splits[B->nbc];
    if (tr ? (mA != nB || nA != mB) : (mA != mB || nA != nB))
        return report_error(COSTA_ERR_SHAPE, "dims(A) != dims(op(B))");
    for (int k = 0; k < A->pr * A->pc; ++k)
        if (A->grid[k] < 0 || A->grid[k] >= P) return report_error(COSTA_ERR_LAYOUT, "A: grid rank out of range");
    for (int k = 0; k < B->pr * B->pc; ++k)
        if (B->grid[k] < 0 || B->grid[k] >= P) return report_error(COSTA_ERR_LAYOUT, "B: grid rank out of range");
    // op(B)'s row axis is B's column axis when transposed
    const int64_t *SBr = tr ? B->col_splits : B->row_splits;
    const int *PBr = tr ? B->col_procs : B->row_procs;
    const int nBr = tr ? B->nbc : B->nbr, npBr = tr ? B->pc : B->pr;
    const int64_t *SBc = tr ? B->row_splits : B->col_splits;
    const int *PBc = tr ? B->row_procs : B->col_procs;
    const int nBc = tr ? B->nbr : B->nbc, npBc = tr ? B->pr : B->pc;
    std::vector<int64_t> rows(static_cast<size_t>(npBr) * A->pr, 0), cols(static_cast<size_t>(npBc) * A->pc, 0);
    if (mA > 0 && nA > 0) {
        axis_overlap(A->row_splits, A->row_procs, A->nbr, A->pr, SBr, PBr, nBr, mA, rows);
        axis_overlap(A->col_splits, A->col_procs, A->nbc, A->pc, SBc, PBc, nBc, nA, cols);
    }
    std::memset(V, 0, sizeof(int64_t) * static_cast<size_t>(P) * P);
    for (int br = 0; br < npBr; ++br)
        for (int bc = 0; bc < npBc; ++bc) {
            // the source process (br, bc) in op(B)'s frame is B's grid (br, bc) or (bc, br)
            const int p = tr ? B->grid[bc * B->pc + br] : B->grid[br * B->pc + bc];
            for (int ar = 0; ar < A->pr; ++ar) {
                const int64_t r = rows[static_cast<size_t>(br) * A->pr + ar];
                if (!r) continue;
                for (int ac = 0; ac < A->pc; ++ac) {
                    const int64_t c = cols[static_cast<size_t>(bc) * A->pc + ac];
                    if (c) V[static_cast<int64_t>(p) * P + A->grid[ar * A->pc + ac]] += r * c;
                }
            }
        }
    return COSTA_OK;
}

extern "C" costa_status costa_grid_block_cyclic(int64_t m, int64_t n, int64_t mb, int64_t nb, int pr, int pc,
                                                char grid_order, const int *rank_perm, int64_t *row_splits,
                                                int *row_procs, int64_t *col_splits, int *col_procs, int *grid,
                                                int *nbr, int *nbc) {
    using costa::report_error;
    if (!nbr || !nbc) return report_error(COSTA_ERR_INVALID_ARG, "costa_grid_block_cyclic: null count");
    if (m < 0 || n < 0 || mb < 1 || nb < 1 || pr < 1 || pc < 1)
        return report_error(COSTA_ERR_INVALID_ARG, "costa_grid_block_cyclic: bad sizes");
    if (grid_order != 'R' && grid_order != 'C')
        return report_error(COSTA_ERR_INVALID_ARG, "costa_grid_block_cyclic: grid_order must be 'R' or 'C'");
    const int64_t br = (m + mb - 1) / mb, bc = (n + nb - 1) / nb;
    if (br > (int64_t(1) << 30) || bc > (int64_t(1) << 30))
        return report_error(COSTA_ERR_INVALID_ARG, "costa_grid_block_cyclic: too many blocks");
    *nbr = static_cast<int>(br);
    *nbc = static_cast<int>(bc);
    if (!row_splits) return COSTA_OK;
    if (!row_procs || !col_splits || !col_procs || !grid)
        return report_error(COSTA_ERR_INVALID_ARG, "costa_grid_block_cyclic: null array");
    const int P = pr * pc;
    if (rank_perm) {
        std::vector<char> seen(P, 0);
        for (int r = 0; r < P; ++r) {
            if (rank_perm[r] < 0 || rank_perm[r] >= P || seen[rank_perm[r]])
                return report_error(COSTA_ERR_INVALID_ARG, "costa_grid_block_cyclic: rank_perm is not a permutation");
            seen[rank_perm[r]] = 1;
        }
    }
    for (int64_t i = 0; i <= br; ++i) row_splits[i] = std::min<int64_t>(i * mb, m);
    for (int64_t j = 0; j <= bc; ++j) col_splits[j] = std::min<int64_t>(j * nb, n);
    for (int64_t i = 0; i < br; ++i) row_procs[i] = static_cast<int>(i % pr);
    for (int64_t j = 0; j < bc; ++j) col_procs[j] = static_cast<int>(j % pc);
    for (int i = 0; i < pr; ++i)
        for (int j = 0; j < pc; ++j) {
            const int r = grid_order == 'R' ? i * pc + j : i + j * pr;
            grid[i * pc + j] = rank_perm ? rank_perm[r] : r;
        }
    return COSTA_OK;
}
