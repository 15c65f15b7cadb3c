"""Parity of the CUDA path (through the C ABI) with the CPU oracle.

Small seeded problems are compared element by element over whole buffers:
bit-exact where the arithmetic allows it (beta = 0, or power-of-two scalars),
otherwise within the tolerance derived in tests/_util.tolerance; padding and
guard elements must stay untouched.  Volumes and relabelings are compared
exactly.
"""
import numpy as np
import pytest

import oracle
from tests._gpu import OnDevice, compare
from workloads import configs as C
from workloads import layouts as L

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def dev():
    d = torch.device("cuda:0")
    torch.cuda.set_device(d)
    return d


def check_problem(p, dev, mode="direct", relabel=True, guard=0):
    g = OnDevice(p, dev, guard=guard)
    try:
        sigma = g.run(relabel=relabel, mode=mode)
        got = g.Ad.download()
        want = g.oracle_result()
        compare(p, got, want, g.Ah, g.Bh)
        # B is read-only
        assert np.array_equal(g.Bd.download().arena, g.Bh.arena, equal_nan=True)
        return sigma, got
    finally:
        g.close()


@pytest.mark.parametrize("case", range(120))
def test_fuzz_direct(case, dev):
    check_problem(C.fuzz_problem(case), dev, guard=3 if case % 4 == 0 else 0)


@pytest.mark.parametrize("case", range(96))
def test_small_blocks(case, dev):
    """Small and odd blocks: the small-tile kernel's pieces and groups, in
    direct and message mode (the two agree bit for bit)."""
    p = C.small_block_problem(case)
    _, direct = check_problem(p, dev)
    _, msg = check_problem(p, dev, mode="message")
    assert np.array_equal(msg.arena, direct.arena, equal_nan=True)
    if case % 3 == 0:  # guard elements around every buffer stay untouched
        check_problem(p, dev, guard=2)


@pytest.mark.parametrize("case", range(120, 180))
def test_fuzz_message_equals_direct(case, dev):
    p = C.fuzz_problem(case)
    _, direct = check_problem(p, dev, mode="direct")
    for relabel in (False, True):
        _, msg = check_problem(p, dev, mode="message", relabel=relabel)
        assert np.array_equal(msg.arena, direct.arena, equal_nan=True)


@pytest.mark.parametrize("dtype", ["f32", "f64", "c64", "c128"])
@pytest.mark.parametrize("op", ["N", "T", "C"])
def test_all_dtypes_ops_multi_tile(dtype, op, dev):
    """Several tiles in each direction plus a ragged tail, both storage orders."""
    for storage_b, storage_a in (("C", "C"), ("R", "C"), ("C", "R"), ("R", "R")):
        m, n = 133, 97
        B = L.block_cyclic(m, n, 40, 24, 2, 3, storage=storage_b, ld_pad=1)
        am, an = (m, n) if op == "N" else (n, m)
        A = L.block_cyclic(am, an, 33, 64, 3, 2, grid_order="C", storage=storage_a)
        for alpha, beta in ((1.0, 0.0), (2.0, 0.5), (-0.3, 0.7)):
            p = C.Problem("grid", dtype, op, alpha, beta, A, B, "uniform",
                          "nan" if beta == 0 else "uniform", C.SEED0 + 9)
            check_problem(p, dev)


def test_c1_bit_exact_and_relabel(dev):
    p = C.c1()
    sigma, _ = check_problem(p, dev, relabel=True, guard=5)
    V = oracle.volume(p.op, p.A, p.B, 4)
    assert oracle.objective(V, sigma) == oracle.lap_optimum(V) == 16384
    assert sigma.tolist() == [0, 1, 2, 3]         # all ties: identity kept


@pytest.mark.parametrize("case", range(30))
def test_volume_matches_oracle(case, dev):
    import paper_2106_06601_gb300 as costa
    p = C.fuzz_problem(case)
    g = OnDevice(p, dev)
    try:
        V = costa.costa_volume(g.LA, g.LB, p.op, torch.cuda.current_stream().cuda_stream)
        assert np.array_equal(V, oracle.volume(p.op, p.A, p.B, p.A.nranks))
        st = costa.costa_plan_stats_get(g.LA, g.LB, p.op, relabel=True)
        assert st["total_volume"] == p.A.m * p.A.n
        assert st["local_identity"] == int(np.trace(V))
        assert st["local_relabeled"] == oracle.lap_optimum(V)
    finally:
        g.close()


def test_relabel_does_not_change_result(dev):
    for case in (5, 17, 33):
        p = C.fuzz_problem(case)
        _, a = check_problem(p, dev, relabel=False)
        _, b = check_problem(p, dev, relabel=True)
        assert np.array_equal(a.arena, b.arena, equal_nan=True)


def test_repeat_calls_deterministic(dev):
    p = C.fuzz_problem(44, dtype="c128")
    p.alpha, p.beta = complex(0.3, -0.2), complex(1.1, 0.4)
    g = OnDevice(p, dev)
    try:
        g.run()
        first = g.Ad.download().arena.copy()
        g.reset_A()
        g.run()
        assert np.array_equal(first, g.Ad.download().arena)
    finally:
        g.close()


def test_edge_cases(dev):
    # 1 x 1, P = 1
    B = L.block_cyclic(1, 1, 1, 1, 1, 1)
    A = L.block_cyclic(1, 1, 4, 4, 1, 1)
    check_problem(C.Problem("1x1", "f64", "T", 2.0, 0.0, A, B, "uniform", "nan"), dev)
    # a single tall column and a single wide row
    for (m, n) in ((1000, 1), (1, 777)):
        B = L.block_cyclic(m, n, 7, 5, 2, 1)
        A = L.block_cyclic(n, m, 3, 11, 1, 2, storage="R")
        check_problem(C.Problem("thin", "f32", "T", 1.0, 0.0, A, B, "uniform", "nan"), dev)
    # empty blocks inside irregular splits
    rs = np.array([0, 0, 5, 5, 17, 40], np.int64)
    cs = np.array([0, 9, 9, 30], np.int64)
    own = np.arange(15, dtype=np.int32).reshape(5, 3) % 4
    A = L.packed_blocks(rs, cs, own, 4)
    B = L.block_cyclic(40, 30, 6, 4, 2, 2)
    check_problem(C.Problem("empty-blocks", "c64", "N", 0.5, -1.0, A, B, "uniform", "uniform"),
                  dev)


def test_empty_matrix(dev):
    import paper_2106_06601_gb300 as costa
    A = L.packed_blocks([0], [0, 5], np.zeros((0, 1), np.int32), 2)
    B = L.packed_blocks([0, 5], [0], np.zeros((1, 0), np.int32), 2)
    LA = costa.costa_layout_create("f64", 2, A.rsplit, A.csplit, A.owner, np.zeros((0, 1)),
                                   A.ld, A.order)
    LB = costa.costa_layout_create("f64", 2, B.rsplit, B.csplit, B.owner, np.zeros((1, 0)),
                                   B.ld, B.order)
    sigma = costa.costa_transform(LA, LB, "T", 1.0, 0.0, relabel=True)
    assert sigma.tolist() == [0, 1]
    assert costa.costa_volume(LA, LB, "T").sum() == 0


def test_batched_matches_oracle(dev):
    import paper_2106_06601_gb300 as costa
    probs = []
    scal = [(1.0, 0.0), (2.0, 0.5), (-0.3, 0.7), (1.0, 0.0), (0.5, 0.0)]
    for k in range(10):
        p = C.fuzz_problem(300 + k, dtype="f64", P=4)
        p.alpha, p.beta = scal[k % len(scal)]
        p.a_kind = "nan" if p.beta == 0 else "uniform"
        probs.append(p)
    gs = [OnDevice(p, dev) for p in probs]
    try:
        stream = torch.cuda.current_stream().cuda_stream
        sigma = costa.costa_transform_batched([g.LA for g in gs], [g.LB for g in gs],
                                              [p.op for p in probs], [p.alpha for p in probs],
                                              [p.beta for p in probs], relabel=True,
                                              stream=stream)
        torch.cuda.synchronize()
        Vsum = sum(oracle.volume(p.op, p.A, p.B, 4) for p in probs)
        assert oracle.objective(Vsum, sigma) == oracle.lap_optimum(Vsum)
        for p, g in zip(probs, gs):
            compare(p, g.Ad.download(), g.oracle_result(), g.Ah, g.Bh)
        # message mode of the same batch gives the same bits
        results = [g.Ad.download().arena.copy() for g in gs]
        for g in gs:
            g.reset_A()
        costa.costa_transform_batched([g.LA for g in gs], [g.LB for g in gs],
                                      [p.op for p in probs], [p.alpha for p in probs],
                                      [p.beta for p in probs], relabel=True, stream=stream,
                                      mode="message")
        torch.cuda.synchronize()
        for g, r in zip(gs, results):
            assert np.array_equal(g.Ad.download().arena, r, equal_nan=True)
    finally:
        for g in gs:
            g.close()


@pytest.mark.parametrize("dtype", ["f64", "c128", "f32"])
@pytest.mark.parametrize("beta", [0.5, 2.0, -0.25, 1.0, 2.0 ** -1000])
def test_special_values_power_of_two_beta(dtype, beta, dev):
    """beta * a formed on the integer pipes must equal the multiply for zeros,
    subnormals, infinities and NaNs, and when beta * a underflows below the
    normal range.  (Values stay below max/4 so that alpha * b and beta * a do
    not overflow: the kernel rounds beta * a before its fma, and an overflow
    there is that formula's result, not the exact one.)"""
    if dtype == "f32" and beta == 2.0 ** -1000:
        pytest.skip("beta is not representable in float")
    rng = np.random.default_rng(5)
    B = L.block_cyclic(64, 48, 16, 16, 2, 2)
    A = L.block_cyclic(48, 64, 8, 32, 2, 2, storage="C")
    p = C.Problem("special", dtype, "T", 2.0, beta, A, B, "uniform", "uniform", C.SEED0)
    g = OnDevice(p, dev)
    try:
        real = np.float64 if dtype in ("f64", "c128") else np.float32
        fi = np.finfo(real)
        specials = np.array([0.0, -0.0, fi.tiny, -fi.tiny, fi.tiny / 4, -fi.smallest_subnormal,
                             fi.max / 4, -fi.max / 5, np.inf, -np.inf, np.nan, 1.5, -3.0,
                             fi.tiny * 2, fi.max / 8, 1e-300 if real is np.float64 else 1e-30],
                            dtype=real)
        for h in (g.Ah, g.Bh):
            v = h.arena.view(real) if dtype in ("c128",) else h.arena.view(real)
            idx = rng.integers(0, v.size, v.size // 3)
            v[idx] = specials[rng.integers(0, specials.size, idx.size)]
        g.Bd.upload(g.Bh)
        g.Ad.upload(g.Ah)
        g.run(relabel=False)
        got = g.Ad.download()
        want = g.oracle_result()
        if np.frexp(abs(beta))[0] == 0.5:
            ok = (got.arena == want.arena) | (np.isnan(got.arena) & np.isnan(want.arena))
            assert np.all(ok), (np.flatnonzero(~ok)[:5], got.arena[~ok][:5], want.arena[~ok][:5])
    finally:
        g.close()


@pytest.mark.parametrize("dtype", ["f64", "c128", "f32"])
@pytest.mark.parametrize("alpha", [2.0, -1.0, 0.25, -(2.0 ** -1000), 2.0 ** 1000])
def test_special_values_power_of_two_alpha(dtype, alpha, dev):
    """alpha * b with beta = 0 and alpha = +-2^k is exact wherever it stays
    in range: the scale kind must equal the oracle bit for bit, with zeros,
    subnormals, infinities and NaNs among the inputs and products that
    underflow below the normal range or overflow."""
    if dtype == "f32" and abs(alpha) in (2.0 ** -1000, 2.0 ** 1000):
        pytest.skip("alpha is not representable in float")
    rng = np.random.default_rng(6)
    B = L.block_cyclic(64, 48, 16, 16, 2, 2)
    A = L.block_cyclic(48, 64, 8, 32, 2, 2, storage="C")
    p = C.Problem("special-a", dtype, "T", alpha, 0.0, A, B, "uniform", "nan", C.SEED0)
    g = OnDevice(p, dev)
    try:
        real = np.float64 if dtype in ("f64", "c128") else np.float32
        fi = np.finfo(real)
        specials = np.array([0.0, -0.0, fi.tiny, -fi.tiny, fi.tiny / 4, -fi.smallest_subnormal,
                             fi.max / 4, -fi.max, np.inf, -np.inf, np.nan, 1.5, -3.0,
                             fi.tiny * 2, fi.max / 8, 1e-300 if real is np.float64 else 1e-30],
                            dtype=real)
        v = g.Bh.arena.view(real)
        idx = rng.integers(0, v.size, v.size // 3)
        v[idx] = specials[rng.integers(0, specials.size, idx.size)]
        g.Bd.upload(g.Bh)
        g.run(relabel=False)
        got, want = g.Ad.download(), g.oracle_result()
        ok = (got.arena == want.arena) | (np.isnan(got.arena) & np.isnan(want.arena))
        assert np.all(ok), (np.flatnonzero(~ok)[:5], got.arena[~ok][:5], want.arena[~ok][:5])
    finally:
        g.close()


def test_phase_timing(dev):
    """Phase events: one phase in direct mode, pack/local/unpack in message
    mode; results are unchanged by the timing; a call with no tiles leaves
    nothing to read."""
    import paper_2106_06601_gb300 as costa
    p = C.fuzz_problem(11, dtype="f64", P=4)
    g = OnDevice(p, dev)
    costa.costa_phase_timing(True)
    try:
        g.run(mode="direct")
        d = costa.costa_phase_times()
        assert len(d) == 1 and d[0] > 0
        want = g.oracle_result()
        compare(p, g.Ad.download(), want, g.Ah, g.Bh)
        g.reset_A()
        g.run(mode="message")
        m = costa.costa_phase_times()
        assert len(m) == 3 and min(m) >= 0 and sum(m) > 0
        compare(p, g.Ad.download(), want, g.Ah, g.Bh)
        # an empty matrix records no phases
        A = L.packed_blocks([0], [0, 5], np.zeros((0, 1), np.int32), 2)
        B = L.packed_blocks([0, 5], [0], np.zeros((1, 0), np.int32), 2)
        LA = costa.costa_layout_create("f64", 2, A.rsplit, A.csplit, A.owner, np.zeros((0, 1)),
                                       A.ld, A.order)
        LB = costa.costa_layout_create("f64", 2, B.rsplit, B.csplit, B.owner, np.zeros((1, 0)),
                                       B.ld, B.order)
        costa.costa_transform(LA, LB, "T", 1.0, 0.0)
        with pytest.raises(costa.CostaError):
            costa.costa_phase_times()
        LA.destroy()
        LB.destroy()
    finally:
        costa.costa_phase_timing(False)
        g.close()


def test_transform_replays_in_cuda_graph(dev):
    """Once its plan exists, a transform call only enqueues kernels on the
    caller's stream, so it can be captured in a CUDA graph and replayed; the
    replays give the oracle's result (for beta != 0 each replay reads the A
    left by the previous one)."""
    import paper_2106_06601_gb300 as costa
    p = C.fuzz_problem(12, dtype="f64", P=4)
    p.alpha, p.beta = 2.0, 0.5
    g = OnDevice(p, dev)
    try:
        s = torch.cuda.Stream(dev)
        costa.costa_transform(g.LA, g.LB, p.op, p.alpha, p.beta, relabel=True, stream=s.cuda_stream)
        torch.cuda.synchronize(dev)
        g.reset_A()
        torch.cuda.synchronize(dev)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=s):
            costa.costa_transform(g.LA, g.LB, p.op, p.alpha, p.beta, relabel=True,
                                  stream=torch.cuda.current_stream().cuda_stream)
        # capture records without running: A is unchanged until the replays
        want = g.Ah.copy()
        for _ in range(3):
            graph.replay()
            torch.cuda.synchronize(dev)
            import oracle
            oracle.transform(p.dtype, p.op, p.alpha, p.beta, p.A, want.buffers(), p.B, g.Bh.buffers())
            got = g.Ad.download()
            ok = (got.arena == want.arena) | (np.isnan(got.arena) & np.isnan(want.arena))
            assert np.all(ok)
    finally:
        g.close()


@pytest.mark.parametrize("dtype", ["f32", "f64", "c64"])
@pytest.mark.parametrize("op", ["N", "T", "C"])
def test_misaligned_runs(dtype, op, dev):
    """Runs off 16-byte boundaries: odd leading dimensions, odd block sizes
    and buffers at odd element offsets (guards).  Copy and scale take the
    16-byte window path, the kinds that read A the element path; both must
    write every element of A once and nothing outside A's blocks."""
    m, n = 150, 171
    am, an = (m, n) if op == "N" else (n, m)
    for k, (pad_b, pad_a, guard) in enumerate(((1, 0, 0), (0, 3, 0), (2, 1, 3), (3, 2, 1))):
        B = L.block_cyclic(m, n, 13 + 2 * k, 37, 2, 3, storage="RC"[k % 2], ld_pad=pad_b)
        A = L.block_cyclic(am, an, 29, 7 + 4 * k, 3, 2, storage="CR"[k % 2], ld_pad=pad_a)
        for alpha, beta in ((1.0, 0.0), (2.0, 0.0), (2.0, 0.5), (-0.3, 0.7)):
            p = C.Problem("misaligned", dtype, op, alpha, beta, A, B, "uniform",
                          "nan" if beta == 0 else "uniform", C.SEED0 + 11 + k)
            check_problem(p, dev, guard=guard)


def _complex_layouts(op):
    """Aligned multi-tile grid with a ragged tail, odd leading dimensions
    (misaligned runs) and 8 x 8 blocks (the small-tile kernel)."""
    m, n = 150, 171
    am, an = (m, n) if op == "N" else (n, m)
    yield L.block_cyclic(m, n, 40, 24, 2, 3), L.block_cyclic(am, an, 33, 64, 3, 2, grid_order="C")
    yield (L.block_cyclic(m, n, 13, 37, 2, 3, storage="R", ld_pad=1),
           L.block_cyclic(am, an, 29, 7, 3, 2, ld_pad=3))
    yield L.block_cyclic(m, n, 8, 8, 2, 3), L.block_cyclic(am, an, 8, 8, 3, 2, grid_order="C")


@pytest.mark.parametrize("dtype", ["c64", "c128"])
@pytest.mark.parametrize("op", ["N", "T", "C"])
@pytest.mark.parametrize("alpha,beta", [(complex(-0.6, 0.3), 0.0),
                                        (complex(0.5, -0.75), 1.0),
                                        (1.0, complex(0.25, 2.0)),
                                        (complex(0.2, 0.9), complex(-1.1, 0.4))])
def test_complex_scalars_within_2ulp(dtype, op, alpha, beta, dev):
    """Complex scalars: each component within 2 ulp(M) of the oracle, M the
    largest of its product terms and of the oracle's value (tests/_util
    tolerance).  A third of A's elements are set to -alpha op(B) / beta, so
    the two halves of each component cancel.  With beta = 0, A is pre-filled
    with NaN and must not be read."""
    from tests._util import global_matrix, max_ulps, op_apply, scatter_global
    for k, (B, A) in enumerate(_complex_layouts(op)):
        p = C.Problem("cplx", dtype, op, alpha, beta, A, B, "uniform",
                      "nan" if beta == 0 else "uniform", C.SEED0 + 40 + k)
        g = OnDevice(p, dev, guard=2)
        try:
            if beta != 0:
                al, be = oracle.scalar(dtype, alpha), oracle.scalar(dtype, beta)
                X = op_apply(op, global_matrix(p.B, g.Bh.buffers())).astype(np.complex128)
                G = global_matrix(p.A, g.Ah.buffers())
                sel = (np.arange(G.size).reshape(G.shape) % 3) == 0
                G[sel] = (-(al * X) / be)[sel].astype(G.dtype)
                scatter_global(p.A, g.Ah.buffers(), G)
                g.Ad.upload(g.Ah)
            g.run()
            got, want = g.Ad.download(), g.oracle_result()
            compare(p, got, want, g.Ah, g.Bh)
            assert np.array_equal(g.Bd.download().arena, g.Bh.arena, equal_nan=True)
            if beta == 0:
                assert not np.isnan(global_matrix(p.A, got.buffers())).any()
            al, be = oracle.scalar(dtype, alpha), oracle.scalar(dtype, beta)
            X = op_apply(op, global_matrix(p.B, g.Bh.buffers()))
            worst = max_ulps(dtype, global_matrix(p.A, got.buffers()),
                             global_matrix(p.A, want.buffers()), al, be, X,
                             global_matrix(p.A, g.Ah.buffers()))
            assert worst <= 2.0, worst
        finally:
            g.close()


@pytest.mark.parametrize("dtype", ["c64", "c128"])
@pytest.mark.parametrize("alpha,beta", [(complex(-0.6, 0.3), 0.0), (complex(0.2, 0.9), complex(-1.1, 0.4))])
def test_special_values_complex_scalars(dtype, alpha, beta, dev):
    """Zeros, subnormals, infinities and NaNs with complex scalars: where the
    plain sum of the rounded products is not finite, both sides return that
    plain IEEE value; elsewhere the 2 ulp(M) bound holds.  (Magnitudes stay
    below max/16, so that no product or partial sum overflows.)"""
    rng = np.random.default_rng(9)
    B = L.block_cyclic(64, 48, 16, 16, 2, 2)
    A = L.block_cyclic(48, 64, 8, 32, 2, 2)
    p = C.Problem("special-c", dtype, "C", alpha, beta, A, B, "uniform", "uniform", C.SEED0)
    g = OnDevice(p, dev)
    try:
        real = np.float64 if dtype == "c128" else np.float32
        fi = np.finfo(real)
        specials = np.array([0.0, -0.0, fi.tiny, -fi.tiny, fi.tiny / 4, -fi.smallest_subnormal,
                             fi.max / 16, -fi.max / 32, np.inf, -np.inf, np.nan, 1.5, -3.0],
                            dtype=real)
        for h in (g.Ah, g.Bh):
            v = h.arena.view(real)
            idx = rng.integers(0, v.size, v.size // 4)
            v[idx] = specials[rng.integers(0, specials.size, idx.size)]
        g.Bd.upload(g.Bh)
        g.Ad.upload(g.Ah)
        g.run(relabel=False)
        compare(p, g.Ad.download(), g.oracle_result(), g.Ah, g.Bh)
    finally:
        g.close()
