"""Grid-like matrix layouts as plain arrays (the input description).

A layout L = (Grid, P, Owners) in the sense of Sec. 5 ("Matrix Layout"):
sorted row splits R and column splits C cut an m x n matrix into blocks
b_ij = rows [R[i], R[i+1]) x cols [C[j], C[j+1]); Owners maps each block to one
of P ranks.  Following the descriptor of Sec. 6 (Fig. 1), each block also
carries its storage: the buffer that holds it, the element offset of its
(0, 0) entry in that buffer, its leading dimension and its element order
(0 = column-major, 1 = row-major).

This module only builds such descriptions and sizes the per-rank buffers.  It
does not intersect layouts, count volumes or move data.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

COL_MAJOR = 0
ROW_MAJOR = 1


@dataclass
class LayoutSpec:
    m: int
    n: int
    rsplit: np.ndarray          # int64 [nbr + 1], non-decreasing, rsplit[0] = 0, rsplit[-1] = m
    csplit: np.ndarray          # int64 [nbc + 1]
    owner: np.ndarray           # int32 [nbr, nbc], values in [0, nranks)
    nranks: int
    buf: np.ndarray             # int32 [nbr, nbc]: storage buffer of each block
    off: np.ndarray             # int64 [nbr, nbc]: element offset of block (0, 0) in its buffer
    ld: np.ndarray              # int64 [nbr, nbc]: leading dimension (elements)
    order: np.ndarray           # int32 [nbr, nbc]: COL_MAJOR or ROW_MAJOR
    bufsize: np.ndarray         # int64 [nbuf]: elements in each buffer
    name: str = ""
    meta: dict = field(default_factory=dict)

    @property
    def nbr(self) -> int:
        return len(self.rsplit) - 1

    @property
    def nbc(self) -> int:
        return len(self.csplit) - 1

    @property
    def nbuf(self) -> int:
        return len(self.bufsize)

    def numel(self) -> int:
        return self.m * self.n

    def check(self) -> None:
        """Consistency of the description itself (not a library check)."""
        assert self.rsplit[0] == 0 and self.rsplit[-1] == self.m
        assert self.csplit[0] == 0 and self.csplit[-1] == self.n
        assert np.all(np.diff(self.rsplit) >= 0) and np.all(np.diff(self.csplit) >= 0)
        for a in (self.owner, self.buf, self.off, self.ld, self.order):
            assert a.shape == (self.nbr, self.nbc)
        assert self.owner.min(initial=0) >= 0 and self.owner.max(initial=0) < self.nranks
        for bi in range(self.nbr):
            h = int(self.rsplit[bi + 1] - self.rsplit[bi])
            for bj in range(self.nbc):
                w = int(self.csplit[bj + 1] - self.csplit[bj])
                if h == 0 or w == 0:
                    continue
                ld = int(self.ld[bi, bj])
                if self.order[bi, bj] == COL_MAJOR:
                    assert ld >= h
                    last = (h - 1) + (w - 1) * ld
                else:
                    assert ld >= w
                    last = (h - 1) * ld + (w - 1)
                assert self.off[bi, bj] >= 0
                assert self.off[bi, bj] + last < self.bufsize[self.buf[bi, bj]]


def _arr(x, dt):
    return np.ascontiguousarray(np.asarray(x, dtype=dt))


def regular_splits(extent: int, bs: int) -> np.ndarray:
    """Splits at multiples of bs; the last block may be partial."""
    s = list(range(0, extent, bs)) + [extent]
    if extent == 0:
        s = [0]
    return _arr(s, np.int64)


def numroc(n: int, nb: int, iproc: int, nprocs: int, isrc: int = 0) -> int:
    """Rows (or columns) of an n-long dimension, blocked by nb and dealt
    cyclically over nprocs processes starting at isrc, held by iproc
    (the ScaLAPACK tool routine NUMROC)."""
    mydist = (nprocs + iproc - isrc) % nprocs
    nblocks = n // nb
    r = (nblocks // nprocs) * nb
    extra = nblocks % nprocs
    if mydist < extra:
        r += nb
    elif mydist == extra:
        r += n % nb
    return r


def block_cyclic(m: int, n: int, mb: int, nb: int, pr: int, pc: int, *,
                 grid_order: str = "R", rank_perm=None, storage: str = "C",
                 ld_pad: int = 0, name: str = "") -> LayoutSpec:
    """ScaLAPACK-style 2D block-cyclic layout with zero source offsets.

    Block (bi, bj) sits on grid process (bi mod pr, bj mod pc); its grid rank
    is pr_i * pc + pc_j ("R") or pr_i + pc_j * pr ("C"); its owner is
    rank_perm[grid rank] (identity if None).  Each rank stores its local
    matrix (numroc rows x numroc cols) in one buffer, column-major with
    LLD = local rows + ld_pad ("C") or row-major with LD = local cols + ld_pad
    ("R").  Local block offsets are (bi div pr) * mb and (bj div pc) * nb.
    """
    P = pr * pc
    perm = list(range(P)) if rank_perm is None else list(rank_perm)
    assert sorted(perm) == list(range(P))
    R, C = regular_splits(m, mb), regular_splits(n, nb)
    nbr, nbc = len(R) - 1, len(C) - 1
    grid_rank = np.empty((pr, pc), dtype=np.int64)
    for i in range(pr):
        for j in range(pc):
            grid_rank[i, j] = i * pc + j if grid_order == "R" else i + j * pr
    loc_rows = [numroc(m, mb, i, pr) for i in range(pr)]
    loc_cols = [numroc(n, nb, j, pc) for j in range(pc)]
    owner = np.empty((nbr, nbc), np.int32)
    off = np.empty((nbr, nbc), np.int64)
    ld = np.empty((nbr, nbc), np.int64)
    bufsize = np.zeros(P, np.int64)
    for i in range(pr):
        for j in range(pc):
            r = perm[grid_rank[i, j]]
            if storage == "C":
                lld = max(1, loc_rows[i]) + ld_pad
                bufsize[r] = lld * loc_cols[j]
            else:
                lld = max(1, loc_cols[j]) + ld_pad
                bufsize[r] = lld * loc_rows[i]
    for bi in range(nbr):
        for bj in range(nbc):
            i, j = bi % pr, bj % pc
            r = perm[grid_rank[i, j]]
            owner[bi, bj] = r
            lr, lc = (bi // pr) * mb, (bj // pc) * nb
            if storage == "C":
                lld = max(1, loc_rows[i]) + ld_pad
                off[bi, bj] = lr + lc * lld
            else:
                lld = max(1, loc_cols[j]) + ld_pad
                off[bi, bj] = lr * lld + lc
            ld[bi, bj] = lld
    order = np.full((nbr, nbc), COL_MAJOR if storage == "C" else ROW_MAJOR, np.int32)
    spec = LayoutSpec(m, n, R, C, owner, P, owner.copy(), off, ld, order, bufsize,
                      name=name or f"bc{mb}x{nb}_{pr}x{pc}{grid_order}",
                      meta=dict(kind="block_cyclic", mb=mb, nb=nb, pr=pr, pc=pc,
                                grid_order=grid_order, storage=storage))
    return spec


def packed_blocks(rsplit, csplit, owner, nranks: int, *, order=None, ld_pad=0,
                  name: str = "") -> LayoutSpec:
    """Arbitrary grid: each rank stores its blocks one after another in its
    buffer (blocks visited in row-major block order), each block dense in its
    own element order with ld = extent + ld_pad."""
    R, C = _arr(rsplit, np.int64), _arr(csplit, np.int64)
    owner = _arr(owner, np.int32)
    nbr, nbc = len(R) - 1, len(C) - 1
    if order is None:
        order = np.zeros((nbr, nbc), np.int32)
    order = _arr(np.broadcast_to(order, (nbr, nbc)), np.int32)
    pad = np.broadcast_to(np.asarray(ld_pad, dtype=np.int64), (nbr, nbc))
    off = np.zeros((nbr, nbc), np.int64)
    ld = np.zeros((nbr, nbc), np.int64)
    cursor = np.zeros(nranks, np.int64)
    for bi in range(nbr):
        h = int(R[bi + 1] - R[bi])
        for bj in range(nbc):
            w = int(C[bj + 1] - C[bj])
            r = int(owner[bi, bj])
            if order[bi, bj] == COL_MAJOR:
                ld[bi, bj] = max(1, h) + int(pad[bi, bj])
                size = ld[bi, bj] * w
            else:
                ld[bi, bj] = max(1, w) + int(pad[bi, bj])
                size = ld[bi, bj] * h
            off[bi, bj] = cursor[r]
            cursor[r] += size
    spec = LayoutSpec(int(R[-1]), int(C[-1]), R, C, owner, nranks, owner.copy(), off,
                      ld, order, cursor.copy(), name=name or "packed",
                      meta=dict(kind="packed"))
    return spec


def row_panels(m: int, n: int, npanels: int, name: str = "") -> LayoutSpec:
    """COSMA-style blocked layout: m rows cut into npanels equal row panels
    (m divisible by npanels); rank k owns panel k, stored column-major with
    ld = panel height, so each panel is one contiguous buffer."""
    assert m % npanels == 0
    h = m // npanels
    R = _arr([k * h for k in range(npanels + 1)], np.int64)
    C = _arr([0, n], np.int64)
    owner = _arr(np.arange(npanels).reshape(npanels, 1), np.int32)
    off = np.zeros((npanels, 1), np.int64)
    ld = np.full((npanels, 1), h, np.int64)
    order = np.zeros((npanels, 1), np.int32)
    bufsize = np.full(npanels, h * n, np.int64)
    return LayoutSpec(m, n, R, C, owner, npanels, owner.copy(), off, ld, order,
                      bufsize, name=name or f"rowpanels{npanels}",
                      meta=dict(kind="row_panels", h=h))


def random_splits(extent: int, nblocks: int, lo: int, hi: int, rng) -> np.ndarray:
    """nblocks sizes in [lo, hi] summing to extent, by rejection sampling:
    draw nblocks-1 sizes uniformly and accept when the remainder is in range."""
    while True:
        sizes = [rng.between(lo, hi) for _ in range(nblocks - 1)]
        last = extent - sum(sizes)
        if lo <= last <= hi:
            sizes.append(last)
            return _arr(np.concatenate([[0], np.cumsum(sizes)]), np.int64)


def scalapack_full(M: int, N: int, MB: int, NB: int, RSRC: int, CSRC: int, pr: int, pc: int,
                   order: str = "R", ld_pad: int = 0):
    """Per-rank local matrix sizes (rows, cols, lld) of a ScaLAPACK
    block-cyclic matrix whose first block sits on process (RSRC, CSRC);
    ranks numbered row-major ("R") or column-major ("C")."""
    out = []
    for rank in range(pr * pc):
        prow, pcol = (rank // pc, rank % pc) if order == "R" else (rank % pr, rank // pr)
        rows = numroc(M, MB, prow, pr, RSRC)
        cols = numroc(N, NB, pcol, pc, CSRC)
        out.append((rows, cols, max(1, rows) + ld_pad))
    return out


def scalapack_sub(M: int, N: int, MB: int, NB: int, RSRC: int, CSRC: int, pr: int, pc: int,
                  order: str, i: int, j: int, m: int, n: int, lld) -> LayoutSpec:
    """The m x n submatrix at 1-based (i, j) of a ScaLAPACK block-cyclic
    matrix as a LayoutSpec over the ranks' local matrices (buffer r = rank
    r's column-major local matrix with leading dimension lld[r]).  Built
    element-wise from the ScaLAPACK index maps: global row g lives on process
    row (g div MB + RSRC) mod pr at local row MB (g div (MB pr)) + g mod MB."""
    g_rows = np.arange(i - 1, i - 1 + m)
    g_cols = np.arange(j - 1, j - 1 + n)
    # blocks of the submatrix: maximal runs of rows (columns) in one global block
    def runs(g, b):
        if len(g) == 0:
            return np.array([0], np.int64)
        blk = g // b
        cut = np.flatnonzero(np.diff(blk)) + 1
        return np.concatenate([[0], cut, [len(g)]]).astype(np.int64)
    R, C = runs(g_rows, MB), runs(g_cols, NB)
    nbr, nbc = len(R) - 1, len(C) - 1
    owner = np.zeros((nbr, nbc), np.int32)
    off = np.zeros((nbr, nbc), np.int64)
    ldm = np.zeros((nbr, nbc), np.int64)
    for bi in range(nbr):
        g = g_rows[R[bi]]
        prow = (g // MB + RSRC) % pr
        lr = MB * (g // (MB * pr)) + g % MB
        for bj in range(nbc):
            h = g_cols[C[bj]]
            pcol = (h // NB + CSRC) % pc
            lc = NB * (h // (NB * pc)) + h % NB
            rank = prow * pc + pcol if order == "R" else prow + pcol * pr
            owner[bi, bj] = rank
            off[bi, bj] = lr + lc * lld[rank]
            ldm[bi, bj] = lld[rank]
    full = scalapack_full(M, N, MB, NB, RSRC, CSRC, pr, pc, order)
    bufsize = np.array([max(1, lld[r]) * max(1, full[r][1]) for r in range(pr * pc)], np.int64)
    return LayoutSpec(m, n, R, C, owner, pr * pc, owner.copy(), off, ldm,
                      np.zeros((nbr, nbc), np.int32), bufsize, name="scalapack_sub",
                      meta=dict(kind="scalapack_sub"))
