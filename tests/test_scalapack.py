"""ScaLAPACK-style interface: submatrix layouts (CPU) and pxgemr2d / pxtran
(GPU) against the oracle.  The tests build each submatrix a second time, in
Python from the ScaLAPACK index maps (workloads.layouts.scalapack_sub)."""
import numpy as np
import pytest

import oracle
from tests._gpu import compare
from workloads import configs as C
from workloads import gen
from workloads import layouts as L
from workloads.materialize import DeviceMatrix, HostMatrix

costa = pytest.importorskip("paper_2106_06601_gb300")

FAKE = 1 << 40


def rand_case(seed):
    rng = gen.IntStream(seed, 61)
    pr, pc = rng.between(1, 3), rng.between(1, 3)
    M, N = rng.between(1, 120), rng.between(1, 120)
    MB, NB = rng.between(1, 17), rng.between(1, 17)
    RSRC, CSRC = rng.below(pr), rng.below(pc)
    order = "RC"[rng.below(2)]
    m, n = rng.between(0, M), rng.between(0, N)
    i, j = rng.between(1, M - m + 1), rng.between(1, N - n + 1)
    pad = rng.below(4)
    full = L.scalapack_full(M, N, MB, NB, RSRC, CSRC, pr, pc, order, ld_pad=pad)
    lld = [f[2] for f in full]
    desc = [1, 0, M, N, MB, NB, RSRC, CSRC, lld[0]]
    return dict(pr=pr, pc=pc, M=M, N=N, MB=MB, NB=NB, RSRC=RSRC, CSRC=CSRC, order=order,
                m=m, n=n, i=i, j=j, lld=lld, desc=desc)


def _fake_grid(c, es):
    ptrs = [FAKE + r * (1 << 32) for r in range(c["pr"] * c["pc"])]
    return costa.BlacsGrid(c["pr"], c["pc"], c["order"], ptrs, c["lld"])


@pytest.mark.parametrize("seed", range(60))
def test_submatrix_layout_matches_index_maps(seed):
    c = rand_case(seed)
    es = 8
    g = _fake_grid(c, es)
    lib_layout = costa.costa_layout_create_scalapack("f64", g, c["i"], c["j"], c["m"], c["n"],
                                                    c["desc"])
    spec = L.scalapack_sub(c["M"], c["N"], c["MB"], c["NB"], c["RSRC"], c["CSRC"], c["pr"],
                           c["pc"], c["order"], c["i"], c["j"], c["m"], c["n"], c["lld"])
    spec.check()
    ptrs = FAKE + spec.buf.astype(np.int64) * (1 << 32) + spec.off * es
    py_layout = costa.costa_layout_from_spec(spec, "f64", ptrs)
    try:
        assert lib_layout.info()[:3] == (c["m"], c["n"], c["pr"] * c["pc"])
        # both describe the same storage: every tile of an N-copy between them
        # reads and writes the same addresses
        t = costa.costa_debug_tiles(lib_layout, py_layout, "N")
        assert np.array_equal(t["src"], t["dst"]) and np.array_equal(t["sld"], t["dld"])
        assert (t["flags"] & 1).sum() == 0
        assert (t["nx"].astype(int) * t["ny"]).sum() == c["m"] * c["n"]
    finally:
        lib_layout.destroy()
        py_layout.destroy()


def test_submatrix_layout_validation():
    c = rand_case(3)
    g = _fake_grid(c, 8)
    for bad_desc, status in (([2] + c["desc"][1:], 1),
                             (c["desc"][:6] + [c["pr"], 0, c["lld"][0]], 1)):
        with pytest.raises(costa.CostaError) as e:
            costa.costa_layout_create_scalapack("f64", g, 1, 1, 1, 1, bad_desc)
        assert e.value.status == status
    with pytest.raises(costa.CostaError) as e:
        costa.costa_layout_create_scalapack("f64", g, c["M"], 1, 2, 1, c["desc"])
    assert e.value.status == 3
    small = costa.BlacsGrid(c["pr"], c["pc"], c["order"],
                            [FAKE] * (c["pr"] * c["pc"]), [0] * (c["pr"] * c["pc"]))
    if c["M"] > 0:
        with pytest.raises(costa.CostaError) as e:
            costa.costa_layout_create_scalapack("f64", small, 1, 1, 1, 1, c["desc"])
        assert e.value.status == 2


# ----------------------------------------------------------------------------
# GPU: pxgemr2d / pxtran against the oracle
# ----------------------------------------------------------------------------

def _matrix(c, dtype, dev, kind, seed, stream0):
    """A full ScaLAPACK matrix: one host and one device arena over the ranks'
    local matrices, plus the submatrix spec and the grid."""
    spec = L.scalapack_sub(c["M"], c["N"], c["MB"], c["NB"], c["RSRC"], c["CSRC"], c["pr"],
                           c["pc"], c["order"], c["i"], c["j"], c["m"], c["n"], c["lld"])
    H = HostMatrix(spec, dtype).fill(kind, seed, lambda r: stream0 + r)
    D = DeviceMatrix(spec, dtype, dev).upload(H)
    ptrs = [D.arena.data_ptr() + int(D.starts[r]) * D.esize for r in range(spec.nbuf)]
    return spec, H, D, costa.BlacsGrid(c["pr"], c["pc"], c["order"], ptrs, c["lld"])


def _pair_cases(seed, transpose):
    rng = gen.IntStream(seed, 71)
    a = rand_case(1000 + seed)
    b = rand_case(2000 + seed)
    # same number of ranks on both grids; sub(B) has sub(A)'s shape (or its transpose)
    b["pr"], b["pc"] = a["pr"] * a["pc"], 1
    if rng.below(2):
        b["pr"], b["pc"] = b["pc"], b["pr"]
    m, n = (a["m"], a["n"]) if not transpose else (a["n"], a["m"])
    b["M"], b["N"] = m + rng.below(9), n + rng.below(9)
    b["RSRC"], b["CSRC"] = rng.below(b["pr"]), rng.below(b["pc"])
    b["m"], b["n"] = m, n
    b["i"], b["j"] = rng.between(1, b["M"] - m + 1), rng.between(1, b["N"] - n + 1)
    full = L.scalapack_full(b["M"], b["N"], b["MB"], b["NB"], b["RSRC"], b["CSRC"], b["pr"],
                            b["pc"], b["order"], ld_pad=rng.below(3))
    b["lld"] = [f[2] for f in full]
    b["desc"] = [1, 0, b["M"], b["N"], b["MB"], b["NB"], b["RSRC"], b["CSRC"], b["lld"][0]]
    return a, b


@pytest.mark.gpu
@pytest.mark.parametrize("seed", range(24))
def test_pxgemr2d_matches_oracle(seed):
    torch = pytest.importorskip("torch")
    dev = torch.device("cuda:0")
    dtype = ("f32", "f64", "c64", "c128")[seed % 4]
    a, b = _pair_cases(seed, transpose=False)
    sa, Ha, Da, ga = _matrix(a, dtype, dev, "uniform", C.SEED0 + 7, 100)
    sb, Hb, Db, gb = _matrix(b, dtype, dev, "uniform", C.SEED0 + 8, 200)
    costa.costa_pxgemr2d(dtype, a["m"], a["n"], ga, a["i"], a["j"], a["desc"], gb, b["i"],
                         b["j"], b["desc"], stream=torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    want = Hb.copy()
    oracle.transform(dtype, "N", 1.0, 0.0, sb, want.buffers(), sa, Ha.buffers())
    p = C.Problem("pxgemr2d", dtype, "N", 1.0, 0.0, sb, sa)
    compare(p, Db.download(), want, Hb, Ha)


@pytest.mark.gpu
@pytest.mark.parametrize("seed", range(24))
def test_pxtran_matches_oracle(seed):
    torch = pytest.importorskip("torch")
    dev = torch.device("cuda:0")
    dtype = ("f32", "f64", "c64", "c128")[seed % 4]
    conj = dtype in ("c64", "c128") and seed % 8 >= 4
    alpha, beta = ((2.0, 0.5), (1.0, 0.0), (-0.3, 0.7))[seed % 3]
    a, c = _pair_cases(seed + 100, transpose=True)
    sa, Ha, Da, ga = _matrix(a, dtype, dev, "uniform", C.SEED0 + 9, 300)
    sc, Hc, Dc, gc = _matrix(c, dtype, dev, "uniform", C.SEED0 + 10, 400)
    costa.costa_pxtran(dtype, c["m"], c["n"], alpha, ga, a["i"], a["j"], a["desc"], beta, gc,
                       c["i"], c["j"], c["desc"], conjugate=conj,
                       stream=torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    op = "C" if conj else "T"
    want = Hc.copy()
    oracle.transform(dtype, op, alpha, beta, sc, want.buffers(), sa, Ha.buffers())
    p = C.Problem("pxtran", dtype, op, alpha, beta, sc, sa)
    compare(p, Dc.download(), want, Hc, Ha)


@pytest.mark.gpu
def test_scalapack_cache_release():
    costa.costa_scalapack_release()
