/*
 * CPU oracle for COSTA's reshuffle A = alpha * op(B) + beta * A, its
 * communication volumes and its optimal process relabeling.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, the package smoke check and the
 * bench's CPU-baseline / reference leg may load this code.  It shares nothing
 * with the CUDA library: no headers, helpers, tables or generators.
 *
 * Everything here follows the plain definitions, element by element:
 *
 *  - transform (Eq. 1, Sec. 5): for every (i, j) of A's index space,
 *      A(i, j) <- alpha * op(B)(i, j) + beta * A(i, j),
 *    op(B)(i, j) = B(i, j) (N), B(j, i) (T) or conj(B(j, i)) (C).  Each element
 *    is located in its layout (Sec. 5 "Matrix Layout", Sec. 6 Fig. 1) by a
 *    binary search in the row and column splits; its storage address is the
 *    block's offset plus r + c*ld (column-major) or r*ld + c (row-major).
 *    When beta == 0, A is not read (BLAS convention), so NaN in A does not
 *    propagate.  Arithmetic: real scalars, beta == 0 give round(alpha * b) in
 *    the data's precision.  Otherwise each real component is the sum of the
 *    exact products rounded once: in double for f32/c64 data (products of
 *    floats are exact in double), and for f64/c128 data by the compensated
 *    dot product Dot2 of Ogita, Rump and Oishi ("Accurate sum and dot
 *    product", SIAM J. Sci. Comput. 26(6), 2005, Alg. 5.3), built on the
 *    error-free TwoSum (Knuth) and TwoProduct (via fma).  This file must be
 *    compiled with -ffp-contract=off and without -ffast-math.
 *
 *  - volume (Sec. 2 "volume", Alg. 2): V[p][q] = number of elements (i, j)
 *    of A whose target block is owned by q and whose source element
 *    op^{-1}(i, j) lies in a block of B owned by p (sender p = owner in L(B),
 *    receiver q = owner in L(A)).  Counted element by element, with no grid
 *    overlay.
 *
 *  - relabeling (Def. COPR, Thm. 1, Remark on the locally-free volume cost):
 *    sigma maximizes sum_q V[sigma(q)][q] over all permutations (sigma(q) is
 *    the process that takes target label q).  Brute force over all P!
 *    permutations in lexicographic order, and an exact dynamic program over
 *    subsets of processes.
 *
 *  - greedy relabeling (Sec. 6, "Max Weight Bipartite Perfect Matching": a
 *    simple greedy algorithm, a 2-approximation): take the pairs (p, q) in
 *    order of decreasing V[p][q] (ties: smaller p first, then smaller q) and
 *    keep a pair when neither p nor q is matched yet; then give the target
 *    labels left over, in increasing order, the processes left over, in
 *    increasing order.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

enum { O_F32 = 0, O_F64 = 1, O_C64 = 2, O_C128 = 3 };
enum { O_N = 0, O_T = 1, O_C = 2 };

/* A layout as plain arrays (Sec. 5 "Matrix Layout"; storage per Sec. 6 Fig. 1). */
typedef struct {
    int64_t nbr, nbc;
    const int64_t *rsplit; /* nbr + 1 */
    const int64_t *csplit; /* nbc + 1 */
    const int32_t *owner;  /* nbr * nbc, block (bi, bj) at bi * nbc + bj */
    const int32_t *buf;    /* storage buffer of each block */
    const int64_t *off;    /* element offset of block (0, 0) in its buffer */
    const int64_t *ld;     /* leading dimension */
    const int32_t *order;  /* 0 column-major, 1 row-major */
} olayout;

/* Index of the block containing coordinate x: the last k with split[k] <= x. */
static int64_t find_block(const int64_t *split, int64_t nb, int64_t x) {
    int64_t lo = 0, hi = nb; /* answer in [lo, hi) */
    while (hi - lo > 1) {
        int64_t mid = lo + (hi - lo) / 2;
        if (split[mid] <= x) lo = mid; else hi = mid;
    }
    /* skip empty blocks that start at the same split value */
    while (lo + 1 < nb && split[lo + 1] <= x) lo++;
    return lo;
}

/* Locate element (i, j): its owner, buffer and element offset. */
void oracle_locate(const olayout *L, int64_t i, int64_t j,
                   int32_t *owner, int32_t *buf, int64_t *off) {
    int64_t bi = find_block(L->rsplit, L->nbr, i);
    int64_t bj = find_block(L->csplit, L->nbc, j);
    int64_t b = bi * L->nbc + bj;
    int64_t r = i - L->rsplit[bi], c = j - L->csplit[bj];
    *owner = L->owner[b];
    *buf = L->buf[b];
    *off = L->off[b] + (L->order[b] == 0 ? r + c * L->ld[b] : r * L->ld[b] + c);
}

void oracle_locate_many(const olayout *L, int64_t n, const int64_t *ij,
                        int32_t *owner, int32_t *buf, int64_t *off) {
    for (int64_t k = 0; k < n; k++)
        oracle_locate(L, ij[2 * k], ij[2 * k + 1], &owner[k], &buf[k], &off[k]);
}

/* ---- error-free transformations and Dot2 (Ogita, Rump, Oishi 2005) ---- */
static void two_sum(double a, double b, double *s, double *e) {
    double x = a + b;
    double z = x - a;
    *e = (a - (x - z)) + (b - z);
    *s = x;
}
static void two_prod(double a, double b, double *p, double *e) {
    double x = a * b;
    *e = fma(a, b, -x);
    *p = x;
}
static double dot2(int n, const double *x, const double *y) {
    double p, s, h, r, q;
    two_prod(x[0], y[0], &p, &s);
    for (int k = 1; k < n; k++) {
        two_prod(x[k], y[k], &h, &r);
        two_sum(p, h, &p, &q);
        s = s + (q + r);
    }
    return p + s;
}

/* Sum of n products of doubles, the exact value rounded (nearly) once.
   Non-finite inputs or an overflowing sum follow plain IEEE evaluation of
   the expression (the error-free transformations would turn inf into NaN). */
static double sum_products(int single, int n, const double *x, const double *y) {
    double plain = 0.0;
    for (int k = 0; k < n; k++) plain += x[k] * y[k];
    if (!isfinite(plain)) return plain;
    if (single) {
        /* float data: products are exact in double, the double sum is within
           2^-53 relative, then one rounding to float by the caller */
        double s = 0.0;
        for (int k = 0; k < n; k++) s += x[k] * y[k];
        return s;
    }
    return dot2(n, x, y);
}

/* out = alpha * b + beta * a for one element; b already conjugated if op = C.
   Values are passed as (re, im) doubles; `single` marks f32/c64 data. */
static void combine(int cplx, int single, const double alpha[2], const double beta[2],
                    const double b[2], const double a[2], double out[2]) {
    int beta0 = (beta[0] == 0.0 && beta[1] == 0.0);
    if (!cplx) {
        if (beta0) {
            out[0] = alpha[0] * b[0];
        } else {
            double x[2] = {alpha[0], beta[0]}, y[2] = {b[0], a[0]};
            out[0] = sum_products(single, 2, x, y);
        }
        out[1] = 0.0;
        return;
    }
    if (alpha[1] == 0.0 && beta[1] == 0.0) {
        /* real scalars: each component independently */
        for (int c = 0; c < 2; c++) {
            if (beta0) {
                out[c] = alpha[0] * b[c];
            } else {
                double x[2] = {alpha[0], beta[0]}, y[2] = {b[c], a[c]};
                out[c] = sum_products(single, 2, x, y);
            }
        }
        return;
    }
    /* complex scalars: re = ar*br - ai*bi + Br*Ar - Bi*Ai,
                        im = ar*bi + ai*br + Br*Ai + Bi*Ar */
    if (beta0) {
        double xr[2] = {alpha[0], -alpha[1]}, yr[2] = {b[0], b[1]};
        double xi[2] = {alpha[0], alpha[1]}, yi[2] = {b[1], b[0]};
        out[0] = sum_products(single, 2, xr, yr);
        out[1] = sum_products(single, 2, xi, yi);
    } else {
        double xr[4] = {alpha[0], -alpha[1], beta[0], -beta[1]};
        double yr[4] = {b[0], b[1], a[0], a[1]};
        double xi[4] = {alpha[0], alpha[1], beta[0], beta[1]};
        double yi[4] = {b[1], b[0], a[1], a[0]};
        out[0] = sum_products(single, 4, xr, yr);
        out[1] = sum_products(single, 4, xi, yi);
    }
}

static void load_elem(int dtype, const void *base, int64_t off, double v[2]) {
    switch (dtype) {
    case O_F32: v[0] = ((const float *)base)[off]; v[1] = 0.0; break;
    case O_F64: v[0] = ((const double *)base)[off]; v[1] = 0.0; break;
    case O_C64: v[0] = ((const float *)base)[2 * off]; v[1] = ((const float *)base)[2 * off + 1]; break;
    default:    v[0] = ((const double *)base)[2 * off]; v[1] = ((const double *)base)[2 * off + 1]; break;
    }
}

static void store_elem(int dtype, void *base, int64_t off, const double v[2]) {
    switch (dtype) {
    case O_F32: ((float *)base)[off] = (float)v[0]; break;
    case O_F64: ((double *)base)[off] = v[0]; break;
    case O_C64: ((float *)base)[2 * off] = (float)v[0]; ((float *)base)[2 * off + 1] = (float)v[1]; break;
    default:    ((double *)base)[2 * off] = v[0]; ((double *)base)[2 * off + 1] = v[1]; break;
    }
}

/* Element-wise combine for values the caller gathered (sampled checks). */
void oracle_combine_many(int dtype, int op, const double *alpha, const double *beta,
                         int64_t n, const void *bvals, const void *avals, void *out) {
    int cplx = (dtype == O_C64 || dtype == O_C128);
    int single = (dtype == O_F32 || dtype == O_C64);
    int beta0 = (beta[0] == 0.0 && beta[1] == 0.0);
    for (int64_t k = 0; k < n; k++) {
        double b[2], a[2] = {0.0, 0.0}, o[2];
        load_elem(dtype, bvals, k, b);
        if (op == O_C && cplx) b[1] = -b[1];
        if (!beta0) load_elem(dtype, avals, k, a);
        combine(cplx, single, alpha, beta, b, a, o);
        store_elem(dtype, out, k, o);
    }
}

/* A <- alpha * op(B) + beta * A for target rows [i_begin, i_end) of A.
   Abufs / Bbufs: host buffers indexed by the layouts' buffer ids.
   Returns 0, or -1 on a shape mismatch. */
int oracle_transform(int dtype, int op, const double *alpha, const double *beta,
                     const olayout *A, void *const *Abufs,
                     const olayout *B, const void *const *Bbufs,
                     int64_t i_begin, int64_t i_end, int nthreads) {
    int64_t mA = A->rsplit[A->nbr], nA = A->csplit[A->nbc];
    int64_t mB = B->rsplit[B->nbr], nB = B->csplit[B->nbc];
    if (op == O_N ? (mA != mB || nA != nB) : (mA != nB || nA != mB)) return -1;
    if (i_begin < 0) i_begin = 0;
    if (i_end > mA) i_end = mA;
    int cplx = (dtype == O_C64 || dtype == O_C128);
    int single = (dtype == O_F32 || dtype == O_C64);
    int beta0 = (beta[0] == 0.0 && beta[1] == 0.0);
#ifdef _OPENMP
    if (nthreads > 0) omp_set_num_threads(nthreads);
#pragma omp parallel for schedule(dynamic, 16)
#endif
    for (int64_t i = i_begin; i < i_end; i++) {
        for (int64_t j = 0; j < nA; j++) {
            int32_t qa, ba, qb, bb;
            int64_t oa, ob;
            oracle_locate(A, i, j, &qa, &ba, &oa);
            if (op == O_N) oracle_locate(B, i, j, &qb, &bb, &ob);
            else oracle_locate(B, j, i, &qb, &bb, &ob);
            double b[2], a[2] = {0.0, 0.0}, o[2];
            load_elem(dtype, Bbufs[bb], ob, b);
            if (op == O_C && cplx) b[1] = -b[1];
            if (!beta0) load_elem(dtype, Abufs[ba], oa, a);
            combine(cplx, single, alpha, beta, b, a, o);
            store_elem(dtype, Abufs[ba], oa, o);
        }
    }
    return 0;
}

/* V[p * P + q] = #elements sent from p (owner in L(B)) to q (owner in L(A)). */
int oracle_volume(int op, const olayout *A, const olayout *B, int P, int64_t *V,
                  int nthreads) {
    int64_t mA = A->rsplit[A->nbr], nA = A->csplit[A->nbc];
    int64_t mB = B->rsplit[B->nbr], nB = B->csplit[B->nbc];
    if (op == O_N ? (mA != mB || nA != nB) : (mA != nB || nA != mB)) return -1;
    memset(V, 0, sizeof(int64_t) * (size_t)P * (size_t)P);
#ifdef _OPENMP
    if (nthreads > 0) omp_set_num_threads(nthreads);
#pragma omp parallel
#endif
    {
        int64_t *loc = (int64_t *)calloc((size_t)P * (size_t)P, sizeof(int64_t));
#ifdef _OPENMP
#pragma omp for schedule(dynamic, 16)
#endif
        for (int64_t i = 0; i < mA; i++) {
            for (int64_t j = 0; j < nA; j++) {
                int32_t qa, ba, qb, bb;
                int64_t oa, ob;
                oracle_locate(A, i, j, &qa, &ba, &oa);
                if (op == O_N) oracle_locate(B, i, j, &qb, &bb, &ob);
                else oracle_locate(B, j, i, &qb, &bb, &ob);
                loc[(int64_t)qb * P + qa] += 1;
            }
        }
#ifdef _OPENMP
#pragma omp critical
#endif
        for (int64_t k = 0; k < (int64_t)P * P; k++) V[k] += loc[k];
        free(loc);
    }
    return 0;
}

/* ---- relabeling: maximize sum_q V[sigma(q)][q] over permutations ---- */

static int next_permutation(int *a, int n) {
    int i = n - 2;
    while (i >= 0 && a[i] >= a[i + 1]) i--;
    if (i < 0) return 0;
    int j = n - 1;
    while (a[j] <= a[i]) j--;
    int t = a[i]; a[i] = a[j]; a[j] = t;
    for (int l = i + 1, r = n - 1; l < r; l++, r--) { t = a[l]; a[l] = a[r]; a[r] = t; }
    return 1;
}

/* All P! permutations in lexicographic order; the first maximum is kept. */
int64_t oracle_lap_bruteforce(int P, const int64_t *V, int *sigma) {
    int perm[16];
    if (P < 1 || P > 12) return INT64_MIN;
    for (int k = 0; k < P; k++) perm[k] = k;
    int64_t best = INT64_MIN;
    do {
        int64_t s = 0;
        for (int q = 0; q < P; q++) s += V[(int64_t)perm[q] * P + q];
        if (s > best) {
            best = s;
            memcpy(sigma, perm, sizeof(int) * (size_t)P);
        }
    } while (next_permutation(perm, P));
    return best;
}

/* Exact DP over subsets: best[S] = best value of giving target labels
   0 .. |S|-1 to the processes in S; label |S|-1 goes to some p in S. */
int64_t oracle_lap_subset_dp(int P, const int64_t *V, int *sigma) {
    if (P < 1 || P > 24) return INT64_MIN;
    size_t nS = (size_t)1 << P;
    int64_t *best = (int64_t *)malloc(nS * sizeof(int64_t));
    int8_t *last = (int8_t *)malloc(nS);
    if (!best || !last) { free(best); free(last); return INT64_MIN; }
    best[0] = 0;
    for (size_t S = 1; S < nS; S++) {
        int q = __builtin_popcountll((unsigned long long)S) - 1;
        int64_t b = INT64_MIN;
        int arg = -1;
        for (int p = 0; p < P; p++) {
            if (!(S >> p & 1)) continue;
            int64_t v = best[S & ~((size_t)1 << p)] + V[(int64_t)p * P + q];
            if (v > b) { b = v; arg = p; }
        }
        best[S] = b;
        last[S] = (int8_t)arg;
    }
    int64_t result = best[nS - 1];
    size_t S = nS - 1;
    for (int q = P - 1; q >= 0; q--) {
        int p = last[S];
        sigma[q] = p;
        S &= ~((size_t)1 << p);
    }
    free(best);
    free(last);
    return result;
}

/* Greedy matching, as described in the header comment. */
int64_t oracle_lap_greedy(int P, const int64_t *V, int *sigma) {
    int64_t n = (int64_t)P * P;
    int64_t *idx = (int64_t *)malloc(sizeof(int64_t) * (size_t)n);
    char *used_p = (char *)calloc((size_t)P, 1), *used_q = (char *)calloc((size_t)P, 1);
    if (!idx || !used_p || !used_q) { free(idx); free(used_p); free(used_q); return INT64_MIN; }
    for (int64_t k = 0; k < n; k++) idx[k] = k;  /* k = p * P + q */
    /* insertion of each pair into the sorted prefix (plain, O(n^2)) */
    for (int64_t i = 1; i < n; i++) {
        int64_t key = idx[i], j = i - 1;
        while (j >= 0) {
            int64_t a = idx[j];
            int before = V[key] > V[a] || (V[key] == V[a] && key < a);
            if (!before) break;
            idx[j + 1] = a;
            j--;
        }
        idx[j + 1] = key;
    }
    for (int q = 0; q < P; q++) sigma[q] = -1;
    for (int64_t i = 0; i < n; i++) {
        int p = (int)(idx[i] / P), q = (int)(idx[i] % P);
        if (!used_p[p] && !used_q[q]) { used_p[p] = used_q[q] = 1; sigma[q] = p; }
    }
    int next_p = 0;
    for (int q = 0; q < P; q++) {
        if (sigma[q] >= 0) continue;
        while (used_p[next_p]) next_p++;
        sigma[q] = next_p;
        used_p[next_p] = 1;
    }
    int64_t total = 0;
    for (int q = 0; q < P; q++) total += V[(int64_t)sigma[q] * P + q];
    free(idx); free(used_p); free(used_q);
    return total;
}

/* Total cost W(G_sigma) of the relabeled communication graph (Def. RG,
   Eq. WG) under the topology cost of Sec. 3: every non-empty package S_ij
   (V[i][j] > 0) is sent from p_i to p_sigma(j) at cost
   w = lat[i][k] + bw[i][k] * V[i][j] with k = sigma(j), or 0 when i == k. */
double oracle_cost_W(int P, const int64_t *V, const double *lat, const double *bw, const int *sigma) {
    double W = 0.0;
    for (int i = 0; i < P; i++)
        for (int j = 0; j < P; j++) {
            int64_t v = V[(int64_t)i * P + j];
            if (v == 0) continue;
            int k = sigma[j];
            if (k == i) continue;
            W += lat[(int64_t)i * P + k] + bw[(int64_t)i * P + k] * (double)v;
        }
    return W;
}

/* COPR by definition (Def. COPR): the permutation of least W(G_sigma), over
   all P! permutations in lexicographic order (the first minimum is kept). */
double oracle_copr_bruteforce_cost(int P, const int64_t *V, const double *lat, const double *bw,
                                   int *sigma) {
    int perm[16];
    if (P < 1 || P > 10) return -1.0;
    for (int k = 0; k < P; k++) perm[k] = k;
    double best = 0.0;
    int first = 1;
    do {
        double W = oracle_cost_W(P, V, lat, bw, perm);
        if (first || W < best) {
            best = W;
            memcpy(sigma, perm, sizeof(int) * (size_t)P);
            first = 0;
        }
    } while (next_permutation(perm, P));
    return best;
}

int oracle_abi_version(void) { return 1; }
