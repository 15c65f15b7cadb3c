"""CPU check of the kernels' index ranges: every tile is the product of a
row piece and a column piece of the plan, and the kernels touch exactly the
tile's elements.  So every access stays inside the tile's A block and its
B block iff every piece lies inside its blocks along its axis and the pieces
tile the axis exactly.  Checked here for every piece of the five workload
configurations and of many random layouts, before any kernel runs."""
import numpy as np
import pytest

from workloads import configs as C
from workloads import layouts as L

costa = pytest.importorskip("paper_2106_06601_gb300")

FAKE = 1 << 40


def _layout(spec, dtype):
    es = {"f32": 4, "f64": 8, "c64": 8, "c128": 16}[dtype]
    ptrs = FAKE + spec.buf.astype(np.int64) * (1 << 32) + spec.off * es
    return costa.costa_layout_from_spec(spec, dtype, ptrs)


def check_pair(p):
    LA, LB = _layout(p.A, p.dtype), _layout(p.B, p.dtype)
    ts = 32  # tile extent of every element type
    try:
        for axis in (0, 1):
            pc = costa.costa_debug_axis_pieces(LA, LB, p.op, axis).astype(np.int64)
            SA = p.A.rsplit if axis == 0 else p.A.csplit
            if p.op == "N":
                SB = p.B.rsplit if axis == 0 else p.B.csplit
            else:
                SB = p.B.csplit if axis == 0 else p.B.rsplit
            extent = SA[-1]
            a_blk, b_blk, a_off, b_off, ln = pc[:, 0], pc[:, 1], pc[:, 2], pc[:, 3], pc[:, 4]
            assert np.all(ln >= 1) and np.all(ln <= ts)
            assert np.all(a_off >= 0) and np.all(b_off >= 0)
            assert np.all(a_off + ln <= SA[a_blk + 1] - SA[a_blk])
            assert np.all(b_off + ln <= SB[b_blk + 1] - SB[b_blk])
            # the pieces cover the axis in order, without gaps or overlap,
            # and both blocks agree on the global position
            start = SA[a_blk] + a_off
            assert np.array_equal(start, SB[b_blk] + b_off)
            assert ln.sum() == extent
            if len(start):
                assert start[0] == 0
                assert np.array_equal(start[1:], start[:-1] + ln[:-1])
    finally:
        LA.destroy()
        LB.destroy()


def check_tiles(p):
    """Every tile's four corners (the tile is affine, so all its addresses lie
    between them) fall inside the source and target rank buffers, the tiles
    cover m * n elements, and the vector flag implies 16-byte alignment."""
    es = {"f32": 4, "f64": 8, "c64": 8, "c128": 16}[p.dtype]
    LA, LB = _layout(p.A, p.dtype), _layout(p.B, p.dtype)
    try:
        t = costa.costa_debug_tiles(LA, LB, p.op)
    finally:
        LA.destroy()
        LB.destroy()
    nx, ny = t["nx"].astype(np.int64), t["ny"].astype(np.int64)
    assert (nx * ny).sum() == p.A.m * p.A.n
    assert np.all(nx >= 1) and np.all(ny >= 1)
    tr = (t["flags"] & 1) != 0
    for name, base, ld, spec, xs, ys in (
            ("dst", t["dst"], t["dld"], p.A, 1, None),
            ("src", t["src"], t["sld"], p.B, None, None)):
        base = base.astype(np.int64)
        ld = ld.astype(np.int64)
        if name == "dst":
            sx, sy = np.ones_like(ld), ld
        else:
            sx = np.where(tr, ld, 1)
            sy = np.where(tr, 1, ld)
        for cx in (0, 1):
            for cy in (0, 1):
                addr = base + ((nx - 1) * cx * sx + (ny - 1) * cy * sy) * es
                rel = addr - FAKE
                buf = rel >> 32
                off = rel - (buf << 32)
                assert np.all(buf >= 0) and np.all(buf < spec.nbuf), name
                assert np.all(off >= 0) and np.all(off < spec.bufsize[buf] * es), name
                assert np.all(off % es == 0), name
    fast = (t["flags"] & 2) != 0
    vec = 16 // es
    assert np.all(t["dst"][fast] % 16 == 0) and np.all(t["src"][fast] % 16 == 0)
    assert np.all((t["dld"][fast].astype(np.int64) * es) % 16 == 0)
    assert np.all((t["sld"][fast].astype(np.int64) * es) % 16 == 0)
    assert np.all(nx[fast] % vec == 0)
    assert np.all(np.where(tr, ny, nx)[fast] % vec == 0)


@pytest.mark.parametrize("name", ["c1", "c2", "c3", "c5"])
def test_config_pieces_in_bounds(name):
    check_pair(C.CONFIGS[name]())
    check_tiles(C.CONFIGS[name]())


def test_c4_pieces_in_bounds():
    for p in C.c4():
        check_pair(p)
        check_tiles(p)


def test_fuzz_pieces_in_bounds():
    for case in range(400):
        check_pair(C.fuzz_problem(case))
        check_tiles(C.fuzz_problem(case))


def _tile_dst(p, rows, cols, u, v):
    """Target address of tile (row piece u, column piece v) from the layout
    spec (independent of the library's tile construction)."""
    es = {"f32": 4, "f64": 8, "c64": 8, "c128": 16}[p.dtype]
    bi, bj = rows[u, 0], cols[v, 0]
    r, c = rows[u, 2].astype(np.int64), cols[v, 2].astype(np.int64)
    A = p.A
    ptr = FAKE + A.buf[bi, bj].astype(np.int64) * (1 << 32) + A.off[bi, bj] * es
    ld = A.ld[bi, bj]
    local = np.where(A.order[bi, bj] == 0, r + c * ld, r * ld + c)
    return (ptr + local * es).astype(np.uint64)


def check_order(p):
    """The kernel's tile order.  Problems whose target tiles are not each
    one contiguous run, of 8- and 16-byte elements (every op) or transposed
    with tiles whose target runs are misaligned holding at least half of the
    elements, walk each target
    buffer in strips of 2 tiles (64 elements for 8-byte and 4-byte
    elements) across its non-contiguous axis, by address inside a strip, one
    target stride group after another; the others follow the global
    super-tile order (k x k pieces, k = 16 for 16-byte elements and 8
    otherwise, row pieces fastest).  Either way the list is a permutation of
    the product of the row and column pieces."""
    es = {"f32": 4, "f64": 8, "c64": 8, "c128": 16}[p.dtype]
    LA, LB = _layout(p.A, p.dtype), _layout(p.B, p.dtype)
    try:
        t = costa.costa_debug_tiles(LA, LB, p.op)
        rows = costa.costa_debug_axis_pieces(LA, LB, p.op, 0)
        cols = costa.costa_debug_axis_pieces(LA, LB, p.op, 1)
    finally:
        LA.destroy()
        LB.destroy()
    nu, nv = len(rows), len(cols)
    if nu * nv == 0:
        assert len(t) == 0
        return
    u, v = np.meshgrid(np.arange(nu), np.arange(nv), indexing="ij")
    u, v = u.ravel(), v.ravel()
    k = 16 if es == 16 else 8
    glob = np.lexsort((u, v, v // k, u // k))  # last key is the primary one
    want = _tile_dst(p, rows, cols, u[glob], v[glob])
    dst = t["dst"].astype(np.uint64)
    assert np.array_equal(np.sort(dst), np.sort(want))
    assert len(np.unique(dst)) == len(dst)
    contiguous = np.all(t["nx"].astype(np.int64) == t["dld"].astype(np.int64))
    area = t["nx"].astype(np.int64) * t["ny"].astype(np.int64)
    a_mis = ((t["dst"] % 16) != 0) | ((t["dld"].astype(np.int64) * es) % 16 != 0) | (t["nx"] % (16 // es) != 0)
    mostly_mis = 2 * area[a_mis].sum() >= area.sum()
    if (es < 8 and (p.op == "N" or not mostly_mis)) or contiguous:
        assert np.array_equal(dst, want)
        return
    ld = t["dld"].astype(np.int64)
    # stride groups are contiguous runs of the list
    change = np.flatnonzero(ld[1:] != ld[:-1]) + 1
    starts = np.concatenate(([0], change))
    ends = np.concatenate((change, [len(ld)]))
    assert len(np.unique(ld[starts])) == len(starts)
    for a, b in zip(starts, ends):
        d = dst[a:b]
        off = ((d - d.min()) // np.uint64(es)).astype(np.int64)
        strip = off // ld[a] // 64
        ds, do = np.diff(strip), np.diff(off)
        assert np.all((ds > 0) | ((ds == 0) & (do > 0)))


@pytest.mark.parametrize("name", ["c1", "c2", "c3", "c5"])
def test_config_tile_order(name):
    check_order(C.CONFIGS[name]())


def test_c4_and_fuzz_tile_order():
    for p in C.c4()[:8]:
        check_order(p)
    for case in range(300):
        check_order(C.fuzz_problem(case))


def _in_buffers(t, spec, es, which):
    """Every access of the tiles `t` on side `which` ("dst" = A, "src" = B)
    falls inside the rank buffers of `spec` (corner test: tiles are affine)."""
    nx, ny = t["nx"].astype(np.int64), t["ny"].astype(np.int64)
    tr = (t["flags"] & 1) != 0
    base = t[which].astype(np.int64)
    ld = (t["dld"] if which == "dst" else t["sld"]).astype(np.int64)
    if which == "dst":
        sx, sy = np.ones_like(ld), ld
    else:
        sx, sy = np.where(tr, ld, 1), np.where(tr, 1, ld)
    for cx in (0, 1):
        for cy in (0, 1):
            rel = base + ((nx - 1) * cx * sx + (ny - 1) * cy * sy) * es - FAKE
            buf = rel >> 32
            off = rel - (buf << 32)
            assert np.all(buf >= 0) and np.all(buf < spec.nbuf), which
            assert np.all(off >= 0) and np.all(off < spec.bufsize[buf] * es), which


def _covered(t, es):
    """Target element addresses covered by the tiles `t`."""
    out = []
    for d in t:
        x = np.arange(int(d["nx"]), dtype=np.int64)
        y = np.arange(int(d["ny"]), dtype=np.int64)
        out.append((int(d["dst"]) + (x[None, :] + y[:, None] * int(d["dld"])) * es).ravel())
    return np.concatenate(out) if out else np.zeros(0, np.int64)


def _pow2(v):
    return 1 << int(np.ceil(np.log2(max(1, v))))


def check_split(p, exact=False):
    """The split between the tile kernel and the small-tile kernel: pieces
    are fast, one warp pass each (every run has its lanes), inside the
    buffers, at most piece_x x piece_y; groups hold at most a full tile's
    passes, of one problem; full-size tiles and pieces together cover A
    exactly once (checked element by element when `exact`)."""
    es = {"f32": 4, "f64": 8, "c64": 8, "c128": 16}[p.dtype]
    vec = 16 // es
    px, py = {4: (16, 8), 8: (8, 8), 16: (8, 4)}[es]
    cap = 32 * 32 * es // 512
    LA, LB = _layout(p.A, p.dtype), _layout(p.B, p.dtype)
    try:
        big, pieces, groups = costa.costa_debug_split(LA, LB, p.op)
        whole = costa.costa_debug_tiles(LA, LB, p.op)
    finally:
        LA.destroy()
        LB.destroy()
    area = lambda t: int((t["nx"].astype(np.int64) * t["ny"].astype(np.int64)).sum())
    assert area(big) + area(pieces) == p.A.m * p.A.n == area(whole)
    # the one-element-per-lane flag: only on misaligned 4-byte tiles whose
    # target runs are off 16-byte boundaries, and on all of those
    assert not np.any(whole["flags"] & 8) and not np.any(pieces["flags"] & 8)
    fast = (big["flags"] & 2) != 0
    elem = (big["flags"] & 8) != 0
    a_mis = ((big["dst"] % 16) != 0) | ((big["dld"].astype(np.int64) * es) % 16 != 0) | (big["nx"] % 4 != 0)
    assert np.array_equal(elem, ~fast & a_mis if es == 4 else np.zeros_like(fast))
    if len(pieces):
        nx, ny = pieces["nx"].astype(np.int64), pieces["ny"].astype(np.int64)
        tr = (pieces["flags"] & 1) != 0
        assert np.all(pieces["flags"] & 2), "pieces take the vector path"
        assert np.all((nx >= 1) & (nx <= px) & (ny >= 1) & (ny <= py))
        assert np.all(nx % vec == 0) and np.all(np.where(tr, ny, nx) % vec == 0)
        lanes_d = np.array([_pow2(v // vec) for v in nx]) * ny
        lanes_s = np.where(tr, nx * np.array([_pow2(v // vec) for v in ny]), lanes_d)
        assert np.all(lanes_d <= 32) and np.all(lanes_s <= 32)
        _in_buffers(pieces, p.A, es, "dst")
        _in_buffers(pieces, p.B, es, "src")
        g = groups.astype(np.int64)
        assert g[0] == 0 and g[-1] == len(pieces)
        sizes = np.diff(g)
        assert np.all(sizes >= 1) and np.all(sizes <= cap)
        for a, b in zip(g[:-1], g[1:]):
            assert len(np.unique(pieces["prob"][a:b])) == 1
    else:
        assert len(groups) == 0
    if exact:
        cov = np.concatenate((_covered(big, es), _covered(pieces, es)))
        assert len(cov) == p.A.m * p.A.n and len(np.unique(cov)) == len(cov)
        assert np.array_equal(np.sort(cov), np.sort(_covered(whole, es)))


@pytest.mark.parametrize("name", ["c1", "c2", "c3", "c5"])
def test_config_split(name):
    check_split(C.CONFIGS[name](), exact=(name == "c1"))


def test_c4_and_fuzz_split():
    for p in C.c4()[:8]:
        check_split(p)
    for case in range(200):
        check_split(C.fuzz_problem(case), exact=True)


def test_small_block_split():
    for case in range(120):
        check_split(C.small_block_problem(case), exact=True)


def test_groups_of_kinds_that_read_a():
    """The second grouping of the pieces (kinds that read A): the same pieces
    in order, one problem per group, at most 8 (f64) or 12 (c64) per group,
    and the copy grouping unchanged for the other types."""
    caps = {"f32": 8, "f64": 8, "c64": 12, "c128": 32}
    seen = set()
    for case in range(96):
        p = C.small_block_problem(case)
        LA, LB = _layout(p.A, p.dtype), _layout(p.B, p.dtype)
        try:
            _, pieces, groups = costa.costa_debug_split(LA, LB, p.op)
            g0 = costa.costa_debug_groups(LA, LB, p.op, False)
            ga = costa.costa_debug_groups(LA, LB, p.op, True)
        finally:
            LA.destroy()
            LB.destroy()
        assert np.array_equal(g0, groups)
        if len(pieces) == 0:
            assert len(ga) == 0
            continue
        ga = ga.astype(np.int64)
        assert ga[0] == 0 and ga[-1] == len(pieces) and np.all(np.diff(ga) >= 1)
        assert np.all(np.diff(ga) <= caps[p.dtype])
        for a, b in zip(ga[:-1], ga[1:]):
            assert len(np.unique(pieces["prob"][a:b])) == 1
        if p.dtype in ("f32", "c128"):
            assert np.array_equal(ga, groups.astype(np.int64))
        seen.add(p.dtype)
    assert {"f64", "c64"} <= seen


_DUMP = """
import hashlib, sys
sys.path.insert(0, %r)
import numpy as np
import paper_2106_06601_gb300 as costa
from workloads import configs as C
from tests.test_plan_bounds import _layout
h = hashlib.sha256()
for p in (C.c3(8192), C.small_blocks(2048), C.c5(rows=16384), C.small_block_problem(4)):
    LA, LB = _layout(p.A, p.dtype), _layout(p.B, p.dtype)
    for part in costa.costa_debug_split(LA, LB, p.op):
        h.update(np.ascontiguousarray(part).tobytes())
    LA.destroy()
    LB.destroy()
print(h.hexdigest())
"""


def test_plan_independent_of_thread_count():
    """Tile lists, their order and the pieces are the same whatever the
    number of planning threads."""
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    out = []
    for t in ("1", "3", "8"):
        env = dict(os.environ, COSTA_PLAN_THREADS=t)
        r = subprocess.run([sys.executable, "-c", _DUMP % root], env=env, capture_output=True, text=True,
                           cwd=root, timeout=600)
        assert r.returncode == 0, r.stderr
        out.append(r.stdout.strip())
    assert out[0] == out[1] == out[2]


def check_halves(p):
    """The x-halves list: each aligned full-size tile at least 32 high and
    wider than 16 along x becomes two tiles (x in [0, 16) and the rest,
    adjacent, on the vector path, inside the buffers); the others stay as
    they are, in order; no halves list for c128, for A blocks longer than
    256 along x, or for op = N with 8-byte elements."""
    es = {"f32": 4, "f64": 8, "c64": 8, "c128": 16}[p.dtype]
    LA, LB = _layout(p.A, p.dtype), _layout(p.B, p.dtype)
    try:
        big, _, _ = costa.costa_debug_split(LA, LB, p.op)
        halves = costa.costa_debug_halves(LA, LB, p.op)
    finally:
        LA.destroy()
        LB.destroy()
    aligned = big[(big["flags"] & 2) != 0]
    rows_fast = p.A.order.flat[0] == L.COL_MAJOR if p.A.order.size else True
    blocks = np.diff(p.A.rsplit if rows_fast else p.A.csplit)
    rule = es in (4, 8) and blocks.max(initial=0) <= 256 and (es == 4 or p.op != "N")
    cut = (aligned["nx"] > 16) & (aligned["ny"] >= 32)
    if not rule or not cut.any():
        assert len(halves) == 0
        return
    assert len(halves) == len(aligned) + int(cut.sum())
    k = 0
    for d, c in zip(aligned, cut):
        if not c:
            assert halves[k].tobytes() == d.tobytes()
            k += 1
            continue
        h0, h1 = halves[k], halves[k + 1]
        k += 2
        tr = bool(d["flags"] & 1)
        assert (h0["nx"], h1["nx"]) == (16, d["nx"] - 16)
        for h in (h0, h1):
            assert (h["ny"], h["dld"], h["sld"], h["prob"], h["flags"]) == \
                   (d["ny"], d["dld"], d["sld"], d["prob"], d["flags"])
            assert h["src"] % 16 == 0 and h["dst"] % 16 == 0
        assert h0["dst"] == d["dst"] and h0["src"] == d["src"]
        assert int(h1["dst"]) == int(d["dst"]) + 16 * es
        assert int(h1["src"]) == int(d["src"]) + (16 * int(d["sld"]) if tr else 16) * es
    _in_buffers(halves, p.A, es, "dst")
    _in_buffers(halves, p.B, es, "src")


def test_halves():
    for name in ("c1", "c2", "c3", "c5"):
        check_halves(C.CONFIGS[name]())
    for p in C.c4()[:8]:
        check_halves(p)
    for case in range(200):
        check_halves(C.fuzz_problem(case))
    # block-cyclic pairs with full tiles: every element type, op and storage,
    # A blocks of 64 and 128 (halves) and 512 (none)
    n_with = 0
    for dt in ("f32", "f64", "c64", "c128"):
        for op in ("N", "T", "C"):
            for k, (amb, st, pad) in enumerate(((64, "C", 0), (128, "R", 2), (512, "C", 1))):
                m, n = 520, 392
                am, an = (m, n) if op == "N" else (n, m)
                B = L.block_cyclic(m, n, 96, 80, 2, 2, storage="CR"[k % 2])
                A = L.block_cyclic(am, an, amb, amb, 2, 2, storage=st, ld_pad=pad)
                p = C.Problem("halves", dt, op, 2.0, 0.5, A, B, "uniform", "uniform", C.SEED0)
                check_halves(p)
                LA, LB = _layout(p.A, p.dtype), _layout(p.B, p.dtype)
                n_with += len(costa.costa_debug_halves(LA, LB, p.op)) > 0
                LA.destroy()
                LB.destroy()
    assert n_with >= 8  # the halves path is exercised
