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
    ptrs = FAKE + (spec.off + spec.buf.astype(np.int64) * (1 << 32)) * es
    return costa.costa_layout_from_spec(spec, dtype, ptrs)


def check_pair(p):
    LA, LB = _layout(p.A, p.dtype), _layout(p.B, p.dtype)
    ts = 16 if p.dtype == "c128" else 32
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


@pytest.mark.parametrize("name", ["c1", "c2", "c3", "c5"])
def test_config_pieces_in_bounds(name):
    check_pair(C.CONFIGS[name]())


def test_c4_pieces_in_bounds():
    for p in C.c4():
        check_pair(p)


def test_fuzz_pieces_in_bounds():
    for case in range(400):
        check_pair(C.fuzz_problem(case))
