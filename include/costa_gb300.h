/*
 * costa_gb300.h: C ABI of a single-GPU (sm_103a) implementation of COSTA's
 * shuffle-and-transpose
 *
 *     A = alpha * op(B) + beta * A,   op in {N (identity), T (transpose),
 *                                           C (conjugate transpose)}       (Eq. 1, Sec. 5)
 *
 * between two grid-like layouts, together with the communication volumes of
 * the reshuffle (Alg. 2) and the communication-optimal process relabeling
 * (COPR, Def. 3 / Thm. 1 / Alg. 1, Sec. 4).
 *
 * The P "processes" of the paper are virtual ranks: a rank is just an owner
 * label, and the blocks it owns live wherever their pointers say (normally
 * one device buffer per rank).  All entry points take plain host or device
 * pointers and sizes; none takes a framework type.
 *
 * Conventions shared by every call:
 *  - Status: each call returns COSTA_OK or an error code, and on error sets a
 *    thread-local message readable with costa_last_error().  All validation
 *    happens before any device work, so a call that fails validation writes
 *    nothing.
 *  - Streams: `stream` is a cudaStream_t passed as void* (NULL = legacy
 *    default stream).  Transform calls are asynchronous on that stream and
 *    return once the kernels are enqueued; the caller keeps every buffer
 *    alive and unmodified until the stream reaches that point.
 *  - Plans: the first transform of a (layouts, op, relabel) combination
 *    builds a plan (grid overlay, volumes, relabeling, tile lists; see
 *    costa_plan_stats) and caches it.  Building a plan synchronizes `stream`.
 *    The TMA-staged tile lists of a plan (real f64 elements, general beta)
 *    are built by the first call of that kind, with synchronous copies; a
 *    call made under stream capture before then uses the cp.async lists.
 *    Plans are freed when one of their layouts is destroyed or by
 *    costa_release_plans().
 *  - Concurrency: every call on one layout pair (A, B) uses the same cached
 *    plan.  The calls that use its device scratch (message mode's staging
 *    buffer; the per-problem scalars of a batch whose scalars differ) run
 *    one after another in call order: a call on another stream than the
 *    previous such call makes its stream wait for that call's completion
 *    event.  Other calls on one pair are not ordered by the library; they
 *    write the same A, so the caller orders them.  Under stream capture the
 *    library adds no wait: the caller orders captured work.  The library's
 *    host state is guarded by one mutex, so calls may come from several
 *    host threads.
 *  - Aliasing: A's and B's storage must not overlap; a layout's blocks must
 *    not overlap each other.  Overlap is not detected and gives undefined
 *    results.
 *  - Arithmetic (Eq. 1): with real alpha and beta each element, or each
 *    component of a complex element, is fma(alpha, b, beta * a) in the
 *    element type's precision (alpha * b when beta == 0, b when also
 *    alpha == 1).  With a complex alpha or beta each component, the sum of
 *    its 2 (beta == 0) or 4 products, is evaluated so that it lies within
 *    2 ulp of the largest product (or of the result, if larger) of the
 *    exactly rounded value: by the compensated dot product Dot2 (Ogita,
 *    Rump & Oishi 2005) for single-precision data; for double-precision
 *    data whose operands are all zero or of magnitude in [2^-480, 2^480),
 *    by an exact fixed-point sum on the integer pipes rounded once (every
 *    four-product component, every other element of two-product ones)
 *    and by Kahan's algorithm for 2 x 2 determinants (the other
 *    two-product ones); Dot2 otherwise.  Repeated calls on one pair give
 *    the same bits.  When beta == 0, A is never read, so NaN or garbage in
 *    A does not propagate.
 */
#ifndef COSTA_GB300_H
#define COSTA_GB300_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    COSTA_OK = 0,
    COSTA_ERR_INVALID_ARG = 1, /* null pointer, bad enum, count out of range */
    COSTA_ERR_LAYOUT = 2,      /* inconsistent layout description            */
    COSTA_ERR_SHAPE = 3,       /* dims(A) != dims(op(B)) or rank counts differ */
    COSTA_ERR_DTYPE = 4,       /* element types of A and B (or of a batch) differ */
    COSTA_ERR_ALLOC = 5,       /* host or device allocation failed           */
    COSTA_ERR_CUDA = 6,        /* a CUDA call failed (message has the error) */
    COSTA_ERR_INTERNAL = 7
} costa_status;

/* Element types: real and complex (interleaved re, im), single and double. */
typedef enum { COSTA_F32 = 0, COSTA_F64 = 1, COSTA_C64 = 2, COSTA_C128 = 3 } costa_dtype;

/* op(B): identity, transpose, conjugate transpose (on real types C == T). */
typedef enum { COSTA_OP_N = 0, COSTA_OP_T = 1, COSTA_OP_C = 2 } costa_op;

/* Element order inside one block (Sec. 6: each block is row- or column-major). */
typedef enum { COSTA_COL_MAJOR = 0, COSTA_ROW_MAJOR = 1 } costa_order;

/* How the data moves on the device:
 *  DIRECT  - one fused kernel reads B's blocks and writes A's blocks
 *            (every pair is treated like a block that stays on its rank, Sec. 6);
 *  MESSAGE - the paper's data flow (Alg. 3, Sec. 6): packages for remote
 *            (source, relabeled target) pairs are packed into one staging
 *            buffer at the exclusive-scan offsets of V, then unpacked and
 *            transformed into A; pairs that are local after relabeling are
 *            remapped directly.  Results are bit-identical to DIRECT. */
typedef enum { COSTA_MODE_DIRECT = 0, COSTA_MODE_MESSAGE = 1 } costa_mode;

/* Storage of one block (Sec. 6, Fig. 1: pointer, stride, ordering).
 *  ptr   - address of the block's (0, 0) element; aligned to the element
 *          size (16 bytes for COSTA_C128).  The block must lie in memory the
 *          current device can address: its own device memory, managed
 *          memory, or host memory allocated or registered with CUDA
 *          (cudaHostAlloc / cudaHostRegister), which the kernels then read
 *          and write directly over the host link.  This is checked when a
 *          plan is built, before any kernel runs (COSTA_ERR_LAYOUT for
 *          pageable host memory, another device's memory or an address
 *          unknown to CUDA).  A source run (a column or row piece of a
 *          block) that does not start or end on a 16-byte boundary may be
 *          read in whole aligned 16-byte chunks: up to 15 bytes before and
 *          after it, in the same aligned chunks (so on the same page), are
 *          read and not used.  Nothing outside A's blocks is written.
 *          NULL marks a block whose rank keeps its storage in another
 *          process (the multi-GPU exchange, costa_exchange_create); calls
 *          that read or write the block reject it with COSTA_ERR_LAYOUT
 *          before any kernel runs.
 *  ld    - leading dimension in elements: the distance between consecutive
 *          columns (column-major) or rows (row-major); ld >= rows
 *          (column-major) or ld >= cols (row-major); ld < 2^31.
 *  order - costa_order. */
typedef struct {
    void *ptr;
    int64_t ld;
    int32_t order;
    int32_t reserved; /* must be 0 */
} costa_block;

typedef struct costa_layout_s *costa_layout;

/* Statistics of a cached plan (volumes in elements). */
typedef struct {
    int64_t total_volume;     /* m * n: elements moved                            */
    int64_t local_identity;   /* trace(V): volume local without relabeling         */
    int64_t local_relabeled;  /* sum_q V[sigma(q)][q]: local volume under sigma     */
    int64_t n_cells;          /* grid-overlay cells (Sec. 5, "Grid Overlay")        */
    int64_t n_tiles;          /* kernel tiles (overlay cells cut to tile size)      */
    int64_t staging_bytes;    /* MESSAGE mode staging size (remote volume x size)   */
    double plan_ms;           /* host + device time to build the plan              */
    double volume_ms;         /* of which: the volume kernel incl. its copy back   */
    double relabel_ms;        /* of which: the assignment solve                    */
} costa_plan_stats;

/* Layout L(A) = (Grid, P, Owners) (Sec. 5, "Matrix Layout") with the block
 * storage of Sec. 6 (Fig. 1).
 *  dt          - element type of the matrix.
 *  nranks      - P >= 1.
 *  nbr, nbc    - block rows / columns (>= 0; 0 gives an empty matrix).
 *  row_splits  - host, nbr + 1 non-decreasing values, row_splits[0] == 0;
 *                block row i holds rows [row_splits[i], row_splits[i+1]);
 *                the matrix has m = row_splits[nbr] rows.  Likewise col_splits.
 *  owners      - host, nbr * nbc ranks in [0, nranks), block (i, j) at i*nbc + j.
 *  blocks      - host, nbr * nbc storage descriptors (same indexing); entries
 *                of empty blocks are ignored.
 * The layout copies all host arrays; device pointers are borrowed.
 * Errors: COSTA_ERR_INVALID_ARG (null pointer, counts), COSTA_ERR_LAYOUT
 * (unsorted splits, owner out of range, ld too small or too large, misaligned
 * block pointer, bad order). */
costa_status costa_layout_create(costa_layout *out, costa_dtype dt, int nranks,
                                 int nbr, const int64_t *row_splits,
                                 int nbc, const int64_t *col_splits,
                                 const int *owners, const costa_block *blocks);

/* ScaLAPACK-style block-cyclic layout (zero source offsets) of an m x n matrix
 * with mb x nb blocks on a pr x pc process grid.  Block (bi, bj) sits on grid
 * process (bi mod pr, bj mod pc), whose grid rank is r = i*pc + j for
 * grid_order 'R' or i + j*pr for 'C'; its owner is rank_perm[r] (identity if
 * rank_perm is NULL).  Each owner o stores its local matrix (NUMROC rows x
 * NUMROC cols) column-major at rank_ptrs[o] with leading dimension lld[o]
 * (>= local rows), so block (bi, bj) starts at local row (bi div pr)*mb and
 * local column (bj div pc)*nb.  rank_ptrs and lld are host arrays of pr*pc
 * entries indexed by owner; a NULL rank_ptrs[o] gives rank o's blocks NULL
 * pointers (storage in another process).  Errors as costa_layout_create. */
costa_status costa_layout_create_block_cyclic(costa_layout *out, costa_dtype dt,
                                              int64_t m, int64_t n, int64_t mb, int64_t nb,
                                              int pr, int pc, char grid_order,
                                              const int *rank_perm,
                                              void *const *rank_ptrs, const int64_t *lld);

/* Frees a layout and every cached plan that uses it.  Synchronizes the
 * device if a plan held device memory.  NULL is accepted. */
costa_status costa_layout_destroy(costa_layout layout);

/* Shape queries. */
costa_status costa_layout_info(costa_layout layout, int64_t *m, int64_t *n,
                               int *nranks, int *dtype);

/* Communication volumes of the reshuffle of B into A's layout (Alg. 2 with
 * the volume V(s) of Sec. 2): V[p * P + q] = number of elements whose source
 * block in L(B) is owned by p and whose target block in L(A) is owned by q.
 * V is a host array of P * P int64.  Runs the overlay/volume kernel on
 * `stream` and synchronizes it.  Errors: INVALID_ARG, SHAPE, CUDA. */
costa_status costa_volume(costa_layout A, costa_layout B, costa_op op, int64_t *V,
                          void *stream);

/* The volumes of costa_volume (same V, same layout of the result) computed
 * without allocating device memory.  The paper has no counterpart: it exists
 * for callers that cannot let a library call cudaMalloc, such as an
 * application whose framework owns all device memory through its own pool,
 * or code on a latency-critical path where cudaMalloc / cudaFree would
 * synchronize the device.
 *  - Memory: all device work happens in one fixed scratch array of 4 MiB
 *    that is part of the library's device image; every GPU that loads the
 *    library holds it until the process exits.  No cudaMalloc, cudaFree or
 *    other allocating call is made, and no plan is built or cached.
 *  - Limit: the pair needs 8 * P^2 bytes for V plus its split and owner
 *    arrays (8 bytes per split, 4 per block of A and of B, each section
 *    rounded up to 256 bytes); more than 4 MiB is rejected with
 *    COSTA_ERR_INVALID_ARG and a message giving both sizes.
 *  - Set-up: every call, with the calling device current, looks up the
 *    array's device address (cudaGetSymbolAddress, which allocates
 *    nothing), so the address stays valid when the device's context is
 *    created again (after cudaDeviceReset).  The first lookup on a device
 *    may load the library's device code: make the first call before any
 *    stream capture.
 *  - Sharing: every call uses the same array, which keeps the last call's
 *    contents (V is zeroed on the stream at the start of each call).  Calls
 *    that overlap on the GPU would race; this entry point is synchronous and
 *    serializes its own calls (also on its error paths, which wait for the
 *    work already queued), so they do not overlap within one process.
 *  - Synchronization: runs on `stream` and synchronizes it before returning.
 * V: host array of P * P int64, as in costa_volume.  Errors: INVALID_ARG,
 * SHAPE, DTYPE, CUDA. */
costa_status costa_volume_noalloc(costa_layout A, costa_layout B, costa_op op, int64_t *V,
                                  void *stream);

/* Communication-optimal process relabeling for the locally-free volume cost
 * (Eq. 2; Remark on the gain and Thm. 1 / Thm. 2, Sec. 4): sigma maximizes
 * sum_q V[sigma[q] * P + q], i.e. target label q is taken by process
 * sigma[q].  Exact, on the host: the Hungarian method (O(P^3)), or for
 * P >= 256 with at most P^2 / 8 nonzero volumes, successive shortest
 * augmenting paths over the nonzero volumes only.  Ties: when the
 * identity attains the optimum the identity is returned.  V: host P * P
 * int64, entries >= 0.  sigma: host, P ints.  local_volume (nullable):
 * receives the optimal sum.  Errors: INVALID_ARG (P < 1, null, negative V). */
costa_status costa_relabel(int P, const int64_t *V, int *sigma, int64_t *local_volume);

/* A = alpha * op(B) + beta * A (Eq. 1, Alg. 3) in COSTA_MODE_DIRECT.
 *  alpha, beta - host pointers to one scalar of the layouts' element type
 *                (float, double, or {re, im} pairs for the complex types).
 *                When beta == 0, A is not read (NaN in A does not propagate).
 *  relabel     - nonzero: compute sigma (costa_relabel on the volumes);
 *                sigma only re-tags target owners, so A's contents are the
 *                same either way.
 *  sigma_out   - nullable host array of P ints; receives sigma (identity when
 *                relabel == 0).
 * Once the plan for (A, B, op) exists, a call only enqueues kernels on
 * `stream`, so it can be captured in a CUDA graph and replayed (build the
 * plan with a first call or costa_plan_stats_get before capturing).
 * Errors: INVALID_ARG, SHAPE (dims(A) != dims(op(B)), P differs), DTYPE,
 * LAYOUT (storage the device cannot address, see costa_block), ALLOC, CUDA. */
costa_status costa_transform(costa_layout A, costa_layout B, costa_op op,
                             const void *alpha, const void *beta, int relabel,
                             int *sigma_out, void *stream);

/* costa_transform with an explicit costa_mode. */
costa_status costa_transform_ex(costa_layout A, costa_layout B, costa_op op,
                                const void *alpha, const void *beta, int relabel,
                                int *sigma_out, costa_mode mode, void *stream);

/* Batched transformation (Sec. 6, "Batched Transformation"): n independent
 * pairs A[k] = alphas[k] * op_k(B[k]) + betas[k] * A[k] in one launch.  All
 * layouts share one element type and one rank count P.  alphas / betas are
 * host arrays of n scalars of that type.  With relabel, one sigma is computed
 * from V summed over the batch (the batch forms one communication round).
 * sigma_out: nullable, P ints. */
costa_status costa_transform_batched(int n, const costa_layout *A, const costa_layout *B,
                                     const costa_op *ops, const void *alphas,
                                     const void *betas, int relabel, int *sigma_out,
                                     void *stream);

/* costa_transform_batched with an explicit costa_mode. */
costa_status costa_transform_batched_ex(int n, const costa_layout *A,
                                        const costa_layout *B, const costa_op *ops,
                                        const void *alphas, const void *betas,
                                        int relabel, int *sigma_out, costa_mode mode,
                                        void *stream);

/* Statistics of the plan for (A, B, op, relabel), building it if needed
 * (which synchronizes `stream`).  For a batch use n > 1 with arrays. */
costa_status costa_plan_stats_get(int n, const costa_layout *A, const costa_layout *B,
                                  const costa_op *ops, int relabel,
                                  costa_plan_stats *stats, void *stream);

/* A process-grid layout described without per-block arrays (for the
 * relabeling study of Sec. 7.2, where blocks can be 1 x 1): block (bi, bj)
 * covers rows [row_splits[bi], row_splits[bi+1]) x columns
 * [col_splits[bj], col_splits[bj+1]) and is owned by rank
 * grid[row_procs[bi] * pc + col_procs[bj]].  Block-cyclic layouts are the
 * case row_procs[bi] = bi mod pr, col_procs[bj] = bj mod pc.  All arrays are
 * host arrays: row_splits nbr + 1, row_procs nbr, col_splits nbc + 1,
 * col_procs nbc, grid pr * pc. */
typedef struct {
    int nbr, nbc;
    const int64_t *row_splits;
    const int *row_procs;
    const int64_t *col_splits;
    const int *col_procs;
    int pr, pc;
    const int *grid;
} costa_grid_desc;

/* Volumes V[p * P + q] of the reshuffle of B into A's layout (as
 * costa_volume, Alg. 2) for process-grid layouts, computed from the 1-D
 * overlaps of the row and column splits: O(blocks per axis + P^2), no
 * overlay cells, no device work.  Errors: INVALID_ARG, LAYOUT, SHAPE. */
costa_status costa_volume_grid(const costa_grid_desc *A, const costa_grid_desc *B, costa_op op, int P,
                               int64_t *V);

/* Fills the arrays of a costa_grid_desc for a block-cyclic m x n layout with
 * mb x nb blocks on a pr x pc grid (zero source offsets; the last block of
 * each axis may be partial): row_splits[i] = min(i * mb, m), row_procs[bi] =
 * bi mod pr, likewise for columns, and grid[i * pc + j] = the rank of grid
 * process (i, j): i * pc + j for grid_order 'R', i + j * pr for 'C', mapped
 * through rank_perm when it is not NULL.  With row_splits == NULL only
 * *nbr and *nbc are written (the array sizes: nbr + 1, nbr, nbc + 1, nbc,
 * pr * pc).  Host only.  Errors: INVALID_ARG. */
costa_status costa_grid_block_cyclic(int64_t m, int64_t n, int64_t mb, int64_t nb, int pr, int pc,
                                     char grid_order, const int *rank_perm, int64_t *row_splits,
                                     int *row_procs, int64_t *col_splits, int *col_procs, int *grid,
                                     int *nbr, int *nbc);

/* The greedy relabeling of Sec. 6 ("a simple greedy algorithm, which is a
 * 2-approximation" of the maximum-weight perfect matching): pairs (p, q) by
 * decreasing V[p * P + q] (ties: smaller p, then smaller q), each kept when p
 * and q are both unmatched; leftover target labels take leftover processes in
 * increasing order.  sigma[q] = p as in costa_relabel; local_volume
 * (nullable) receives sum_q V[sigma[q] * P + q], at least half the optimum.
 * Host only.  Errors: INVALID_ARG. */
costa_status costa_relabel_greedy(int P, const int64_t *V, int *sigma, int64_t *local_volume);

/* Relabeling under a general communication cost (Sec. 3): sending a package
 * of volume v from process i to process j != i costs lat[i * P + j] +
 * bw[i * P + j] * v (network topology: latency and bandwidth cost per element);
 * local packages and empty packages cost nothing.  sigma (sigma[q] = process
 * that takes target label q) minimizes the total cost W(G_sigma) of the
 * relabeled communication graph (Def. COPR, Eq. WG).  Following Alg. 1 it is
 * found as the assignment maximizing the total relabeling gain (Eq. delta,
 * Thm. 1), solved exactly (Hungarian method on doubles, O(P^3)); the identity
 * is kept when it is optimal.  cost_identity / cost_relabeled (nullable)
 * receive W(G) and W(G_sigma).  With lat = 0 and bw = 1 off the diagonal this
 * is costa_relabel's objective.  Host only.  Errors: INVALID_ARG (P < 1,
 * null, negative V, non-finite costs). */
costa_status costa_relabel_cost(int P, const int64_t *V, const double *lat, const double *bw, int *sigma,
                                double *cost_identity, double *cost_relabeled);

/* ---- ScaLAPACK-style interface (Sec. 6: pxgemr2d and pxtran wrappers) ----
 *
 * A BLACS-like process grid of virtual ranks: nprow x npcol processes,
 * numbered row-major ('R': rank = prow * npcol + pcol) or column-major
 * ('C': rank = prow + pcol * nprow).  local[rank] is the device address of
 * that rank's local matrix, column-major with leading dimension lld[rank]
 * (lld NULL: every rank uses the descriptor's LLD). */
typedef struct {
    int nprow, npcol;
    char order;
    void *const *local;
    const int64_t *lld;
} costa_blacs_grid;

/* Layout of the submatrix rows i..i+m-1, columns j..j+n-1 (1-based, as in
 * ScaLAPACK) of a block-cyclic matrix with array descriptor
 * desc = {DTYPE_ = 1, CTXT_ (ignored), M_, N_, MB_, NB_, RSRC_, CSRC_, LLD_}
 * distributed over grid g: the global block grid truncated to the submatrix
 * (Sec. 5), each block pointing into its owner's local matrix at the
 * ScaLAPACK local indices (INDXG2L).  Host only; the layout borrows the local
 * pointers.  Errors: INVALID_ARG, SHAPE (submatrix outside M_ x N_), LAYOUT
 * (LLD below NUMROC rows, null local pointer), DTYPE. */
costa_status costa_layout_create_scalapack(costa_layout *out, costa_dtype dt, const costa_blacs_grid *g,
                                           int64_t i, int64_t j, int64_t m, int64_t n,
                                           const int64_t *desc);

/* sub(B) := sub(A), the m x n submatrices A(ia.., ja..) and B(ib.., jb..)
 * (ScaLAPACK PxGEMR2D).  The two grids must have the same number of ranks.
 * Asynchronous on stream like costa_transform; the first call with a given
 * argument set builds and caches its layouts and plan (32 entries, least
 * recently used evicted). */
costa_status costa_pxgemr2d(costa_dtype dt, int64_t m, int64_t n, const costa_blacs_grid *ga, int64_t ia,
                            int64_t ja, const int64_t *desca, const costa_blacs_grid *gb, int64_t ib,
                            int64_t jb, const int64_t *descb, void *stream);

/* sub(C) := beta * sub(C) + alpha * op(sub(A)), sub(C) m x n, sub(A) n x m,
 * op = transpose (conjugate = 0: PxTRAN / PxTRANU) or conjugate transpose
 * (conjugate != 0: PxTRANC).  alpha, beta: host scalars of dt.  Caching as
 * costa_pxgemr2d. */
costa_status costa_pxtran(costa_dtype dt, int conjugate, int64_t m, int64_t n, const void *alpha,
                          const costa_blacs_grid *ga, int64_t ia, int64_t ja, const int64_t *desca,
                          const void *beta, const costa_blacs_grid *gc, int64_t ic, int64_t jc,
                          const int64_t *descc, void *stream);

/* Frees the layouts (and plans) cached by costa_pxgemr2d / costa_pxtran. */
costa_status costa_scalapack_release(void);

/* ---- Multi-GPU exchange (Sec. 6 "Implementation", Alg. 3) ----
 *
 * The reshuffle with the P ranks placed on G GPUs, one process per GPU:
 * rank r's blocks (of A and of B) live on GPU place[r].  Process g (on GPU
 * g, the current device) runs, for A = alpha * op(B) + beta * A:
 *   costa_exchange_pack    - copies each tile whose source rank is on g and
 *                            whose target rank is on another GPU h into h's
 *                            segment of g's send buffer (exactly: the
 *                            transform comes after the transfer, Sec. 6);
 *   costa_exchange_local   - the tiles with both ranks on g, B -> A directly;
 *   the caller's exchange  - an all-to-all-v of the segments: g's segment for
 *                            h goes to g's segment of h's receive buffer
 *                            (e.g. NCCL grouped send/receive); the library
 *                            never touches another GPU's memory;
 *   costa_exchange_unpack  - each received tile into A with op, alpha, beta.
 * pack and local may run together; unpack needs the whole receive buffer.
 * The result equals costa_transform on one device bit for bit.
 *
 * Every process builds the same tiles from the layouts (splits, owners and
 * storage orders, which must be identical in all processes) in one fixed
 * canonical order, so the package contents and offsets agree without any
 * coordination.  Segments are ordered by peer GPU: segment h starts at the
 * sum of the sizes of segments 0 .. h-1 (the all-to-all-v displacements).
 * Layouts may give NULL pointers for the blocks of ranks on other GPUs
 * (costa_block); the blocks of ranks on g must be addressable by g.
 * Relabeling (costa_relabel_placement) is a planning step before this: the
 * caller moves label q's target blocks to process sigma[q], i.e. builds A's
 * layout with owner sigma[q] in place of q. */
typedef struct costa_exchange_s *costa_exchange;

/* Bytes of g's send segments (send_bytes[h]: to GPU h) and receive segments
 * (recv_bytes[h]: from GPU h); [g] is 0 in both.  Host only.  place: host,
 * P ints in [0, G).  Errors: INVALID_ARG, SHAPE, DTYPE. */
costa_status costa_exchange_sizes(costa_layout A, costa_layout B, costa_op op, int G, const int *place,
                                  int g, int64_t *send_bytes, int64_t *recv_bytes);

/* Builds process g's pack, local and unpack tile lists for the send and
 * receive buffers send_buf and recv_buf (device memory of the current device,
 * 16-byte aligned, of at least the sum of costa_exchange_sizes' send_bytes /
 * recv_bytes; the caller owns them and keeps them alive with the exchange).
 * The exchange owns one device allocation for its tables, freed by
 * costa_exchange_destroy.  Errors: INVALID_ARG (placement, buffers), SHAPE,
 * DTYPE, LAYOUT (a block of a rank on g that g cannot address), ALLOC, CUDA. */
costa_status costa_exchange_create(costa_exchange *out, costa_layout A, costa_layout B, costa_op op, int G,
                                   const int *place, int g, void *send_buf, void *recv_buf);

/* The exchange's segment sizes in bytes (host arrays of G), as
 * costa_exchange_sizes. */
costa_status costa_exchange_counts(costa_exchange x, int64_t *send_bytes, int64_t *recv_bytes);

/* Enqueue the phases on `stream` (asynchronous; the current device must be
 * the exchange's).  alpha, beta: host scalars of the element type, as
 * costa_transform; with beta == 0, A is not read. */
costa_status costa_exchange_pack(costa_exchange x, void *stream);
costa_status costa_exchange_local(costa_exchange x, const void *alpha, const void *beta, void *stream);
costa_status costa_exchange_unpack(costa_exchange x, const void *alpha, const void *beta, void *stream);

costa_status costa_exchange_destroy(costa_exchange x);

/* Relabeling for a placement (Sec. 3 network-topology cost, Def. COPR):
 * sigma minimizes W(G_sigma) where a package of v elements kept on its
 * process costs 0, one between two ranks on the same GPU intra * v, and one
 * between GPUs v (the bytes that cross the GPU link, weighted 1).  Solved
 * as costa_relabel_cost.  cost_identity / cost_relabeled (nullable) receive
 * W(G) and W(G_sigma).  Host only.  Errors: INVALID_ARG. */
costa_status costa_relabel_placement(int P, const int64_t *V, int G, const int *place, double intra, int *sigma,
                                     double *cost_identity, double *cost_relabeled);

/* ---- Housekeeping ---- */

/* Frees every cached plan (synchronizes the device). */
costa_status costa_release_plans(void);

/* Thread-local message of the last failed call on this thread ("" if none). */
const char *costa_last_error(void);

/* ---- Diagnostics ----
 *
 * Not needed to reshuffle: they expose the planner's tile lists (host only,
 * no device work), count kernel launches, and time the phases of transform
 * calls, for tests, tuning and profiling. */

/* Diagnostics (host only, no device work): the pieces into which the plan
 * cuts one axis of A (axis 0 = rows, 1 = columns) for the pair (A, B, op).
 * Each piece is 6 int32: {A block index, op(B) block index, offset in A's
 * block, offset in op(B)'s block, length, overlay interval index}; the
 * kernel's tiles are the products of row pieces and column pieces.  Writes
 * min(*count, cap) pieces to out (6 * cap int32) and the total to *count. */
costa_status costa_debug_axis_pieces(costa_layout A, costa_layout B, costa_op op, int axis,
                                     int32_t *out, int64_t cap, int64_t *count);

/* Diagnostics (host only, no device work): the remap kernel's tile list for
 * (A, B, op) in direct mode, in the order the kernel's warps take the tiles.  Each tile is 32 bytes: {source address, target
 * address (uint64), source stride, target stride (int32), nx, ny, problem,
 * flags (uint16)}, in the frame where x runs along A's contiguous axis
 * (flags: 1 = transposed, 2 = vector path, 4 = conjugate).  Writes
 * min(*count, cap) tiles to out (32 * cap bytes) and the total to *count. */
costa_status costa_debug_tiles(costa_layout A, costa_layout B, costa_op op, void *out, int64_t cap,
                               int64_t *count);

/* Diagnostics (host only, no device work): how the direct tile list of
 * (A, B, op) is split between the two remap kernels.  Tiles needing fewer
 * than half of a full tile's warp passes are cut into pieces of one warp
 * pass each (at most 8 x 8 elements; 16 x 8 for 4-byte and 8 x 4 for
 * 16-byte elements, x along A's contiguous axis), which the small-tile
 * kernel moves in groups of up to a full tile's passes; the other tiles stay
 * with the tile kernel (those whose runs are not 16-byte aligned after the
 * others, for its instance for misaligned tiles).  Writes up to cap_tiles full-size tiles to `tiles`
 * and up to cap_pieces pieces to `pieces` (32-byte descriptors as in
 * costa_debug_tiles), and up to cap_groups group offsets to `groups` (group
 * g covers pieces [groups[g], groups[g + 1]), so there are *ngroups + 1
 * offsets when *ngroups > 0); the totals go to *ntiles, *npieces and
 * *ngroups. */
costa_status costa_debug_split(costa_layout A, costa_layout B, costa_op op, void *tiles, int64_t cap_tiles,
                               void *pieces, int64_t cap_pieces, uint32_t *groups, int64_t cap_groups,
                               int64_t *ntiles, int64_t *npieces, int64_t *ngroups);

/* Diagnostics (host only, no device work): the group offsets over the
 * pieces of costa_debug_split that the small-tile kernel uses for the copy
 * and scale kinds (reads_a = 0) or for the kinds that read A (reads_a != 0:
 * at most 8 pieces per group for f64, 12 for c64, as for copy otherwise).
 * Writes up to cap_groups offsets to `groups` (group g covers pieces
 * [groups[g], groups[g + 1])) and the number of groups to *ngroups. */
costa_status costa_debug_groups(costa_layout A, costa_layout B, costa_op op, int reads_a, uint32_t *groups,
                                int64_t cap_groups, int64_t *ngroups);

/* Diagnostics (host only, no device work): the aligned full-size tiles of
 * (A, B, op) as x-halves, the list that the f32 kinds and the f64 / c64
 * axpby kind with beta = +-2^k run on.  A tile at least 32 high and wider
 * than 16 along A's contiguous axis becomes two tiles, columns [0, 16) and
 * the rest, adjacent in the list; the others stay as they are.  Writes up
 * to cap_tiles 32-byte descriptors (as in costa_debug_tiles) to `tiles` and
 * the total to *ntiles, which is 0 when the pair has no halves list: 16-byte
 * elements, A blocks longer than 256 along A's contiguous axis, op = N with
 * 8-byte elements, or no tile to cut. */
costa_status costa_debug_halves(costa_layout A, costa_layout B, costa_op op, void *tiles, int64_t cap_tiles,
                                int64_t *ntiles);

/* Diagnostics (host only, no device work): process g's exchange lists for
 * buffers at the addresses send_base / recv_base: which = 0 pack, 1 local,
 * 2 unpack, unsplit, in the canonical order (32-byte descriptors as in
 * costa_debug_tiles).  Writes min(*count, cap) descriptors to out and the
 * total to *count; volumes (nullable, 2 * G int64): the elements of A that g
 * sends to each GPU h, then those it receives from each h. */
costa_status costa_debug_exchange(costa_layout A, costa_layout B, costa_op op, int G, const int *place, int g,
                                  uint64_t send_base, uint64_t recv_base, int which, void *out, int64_t cap,
                                  int64_t *count, int64_t *volumes);

/* Diagnostics: TMA staging of the tile kernel's source tiles.  By default
 * (environment variable COSTA_TMA unset when a plan is built) only f64 data
 * with a beta that is neither 0 nor +-2^k uses it (measured faster there,
 * slower for every other kind and type); COSTA_TMA=0 turns it off and
 * COSTA_TMA=1 on for every kind and type.  Builds the plan of (A, B, op)
 * and its TMA-staged lists if needed (a transform builds them on the first
 * call of a kind that uses them), then writes out[0] = TMA tiles in the
 * direct list, out[1] = in its x-halves list,
 * out[2] = tensor maps, out[3] = TMA waits that gave up in this plan's
 * launches (each ends its warp's work and should never happen), out[4] and
 * out[5] = the kinds (bit per combine kind) that take the TMA tiles of the
 * two lists.  out: host, 6 int64.  Synchronizes the device. */
costa_status costa_debug_tma(costa_layout A, costa_layout B, costa_op op, int64_t *out);

/* Diagnostics (host only, no device work): the fixed-point sum of products
 * that the remap kernels use for each component of alpha * op(B) + beta * A
 * with complex scalars on double complex data (Eq. 1), evaluated on the host
 * by the same code.  For each of `count` sets, out[k] = the sum over
 * i < n of (-1)^neg[k n + i] x[k n + i] * y[k n + i], rounded once to
 * double (within 0.5 ulp of the result plus n * 2^-7 ulp of the largest
 * product of the exact sum); n is 2 or 4.  x, y, neg, out: host arrays.
 * Every factor must be zero or of magnitude in [2^-480, 2^480), the range
 * in which the kernels take this evaluation; COSTA_ERR_INVALID_ARG
 * otherwise, with nothing written. */
costa_status costa_debug_fxdot(int n, int64_t count, const double *x, const double *y, const int32_t *neg,
                               double *out);

/* Number of kernels this library has launched in this process. */
int64_t costa_kernel_launch_count(void);

/* Per-phase device time of transform calls (diagnostic).  While enabled
 * (enable != 0; process-wide, off at load), every costa_transform* call
 * records CUDA events on its stream around its phases: the remap launches in
 * direct mode (1 phase); pack, local remap and unpack in message mode (3
 * phases: Alg. 3 and Sec. 6, packing, the blocks that stay local, unpacking
 * with the transform).  The events add no synchronization to the call. */
costa_status costa_phase_timing(int enable);

/* Waits for the events of the last timed transform call on the calling
 * host thread's current device and writes its phase durations in
 * milliseconds to ms[0 .. *nphases - 1] (ms: host array of 3 doubles).
 * COSTA_ERR_INVALID_ARG if no call has been timed since timing was enabled,
 * or if the last timed call had no tiles. */
costa_status costa_phase_times(double *ms, int *nphases);

/* ABI version of this header (1). */
int costa_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* COSTA_GB300_H */
