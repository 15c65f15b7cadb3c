"""CPU check of the kernels' index ranges: every tile is the product of a
row piece and a column piece of the plan, and the kernels touch exactly the
tile's elements.  So every access stays inside the tile's A block and its
B block iff every piece lies inside its blocks along its axis and the pieces
tile the axis exactly.  Checked here for every piece of the five workload
configurations and of many random layouts, before any kernel runs."""
import numpy as np
import pytest

from workloads import configs as C

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
