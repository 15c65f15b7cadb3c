"""The five workload configurations at full size, in the launch configuration
the bench times (one costa_transform / costa_transform_batched call, direct
mode, cached plan).

Inputs are filled on the device by the seeded generator and read back before
the transform.  Every element of A is then compared with the oracle run over
the whole matrix on the host cores: all of c2-c5 (c4's 64 instances each),
c5b, bc8 and the misaligned workloads ld1 (f32 target with an odd leading
dimension) and odd (odd block sizes) are in the bit-exact class (beta = 0,
or power-of-two alpha and beta).  A sampled check (random points plus block corners and edges) runs
first as a fast pre-check.  B must be bit-for-bit unchanged, compared on the
device with a copy taken before the call.  Volumes and optima are checked
against the hand-derived closed forms (tests/golden/closed_forms.json).
"""
import json
import os

import numpy as np
import pytest

import oracle
from tests._util import assert_close, exact_case
from workloads import configs as C
from workloads.materialize import DeviceMatrix

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "closed_forms.json")


@pytest.fixture(scope="module")
def dev():
    d = torch.device("cuda:0")
    torch.cuda.set_device(d)
    return d


def sample_points(spec, n_random: int, seed: int) -> np.ndarray:
    rng = np.random.default_rng(seed)
    pts = [np.stack([rng.integers(0, spec.m, n_random), rng.integers(0, spec.n, n_random)], 1)]
    # corners and edge midpoints of (up to) 4096 blocks
    nb = spec.nbr * spec.nbc
    pick = rng.choice(nb, size=min(nb, 4096), replace=False)
    bi, bj = pick // spec.nbc, pick % spec.nbc
    r0, r1 = spec.rsplit[bi], spec.rsplit[bi + 1] - 1
    c0, c1 = spec.csplit[bj], spec.csplit[bj + 1] - 1
    ok = (r1 >= r0) & (c1 >= c0)
    for a, b in ((r0, c0), (r0, c1), (r1, c0), (r1, c1), ((r0 + r1) // 2, c1), (r1, (c0 + c1) // 2)):
        pts.append(np.stack([a[ok], b[ok]], 1))
    return np.concatenate(pts).astype(np.int64)


class Mat:
    def __init__(self, p, dev):
        import paper_2106_06601_gb300 as costa
        self.p = p
        self.Bd = DeviceMatrix(p.B, p.dtype, dev).fill(p.b_kind, p.seed, p.src_stream)
        self.Ad = DeviceMatrix(p.A, p.dtype, dev).fill(p.a_kind, p.seed, p.tgt_stream)
        self.LA = costa.costa_layout_from_spec(p.A, p.dtype, self.Ad.block_ptrs())
        self.LB = costa.costa_layout_from_spec(p.B, p.dtype, self.Bd.block_ptrs())

    def sample_index(self, ij):
        _, abuf, aoff = oracle.locate(self.p.A, ij)
        src = ij if self.p.op == "N" else ij[:, ::-1].copy()
        _, bbuf, boff = oracle.locate(self.p.B, src)
        ia = torch.as_tensor(self.Ad.starts[abuf] + aoff, device=self.Ad.arena.device)
        ib = torch.as_tensor(self.Bd.starts[bbuf] + boff, device=self.Bd.arena.device)
        return ia, ib

    def close(self):
        self.LA.destroy()
        self.LB.destroy()


def check_samples(p, a_pre, b, a_post):
    want = oracle.combine(p.dtype, p.op, p.alpha, p.beta, b, a_pre)
    al, be = oracle.scalar(p.dtype, p.alpha), oracle.scalar(p.dtype, p.beta)
    bvals = b.astype(np.complex128)
    if p.op == "C":
        bvals = np.conj(bvals)
    assert_close(p.dtype, a_post, want, al, be,
                 bvals if p.dtype in ("c64", "c128") else bvals.real, a_pre,
                 exact=exact_case(p.dtype, al, be))


def bits(t):
    """An integer view of a tensor's bytes (bitwise comparison)."""
    if t.is_complex():
        t = torch.view_as_real(t)
    return t.view(torch.int64 if t.element_size() == 8 else torch.int32)


def count_mismatches(got: np.ndarray, want: np.ndarray, chunk: int = 1 << 26) -> int:
    """Elements whose values differ (NaN only matches NaN), in chunks to bound
    the temporaries on multi-GB arenas."""
    bad = 0
    for k in range(0, got.size, chunk):
        g, w = got[k:k + chunk], want[k:k + chunk]
        ok = (g == w) | (np.isnan(g) & np.isnan(w))
        bad += int(g.size - np.count_nonzero(ok))
    return bad


def whole_buffer_check(p, a_host, b_host, got_host):
    """a_host (A before the call) becomes the oracle's result in place; every
    arena element of the GPU result must equal it: block elements bit-exact
    (the configs are all in the exact class), padding unchanged."""
    al, be = oracle.scalar(p.dtype, p.alpha), oracle.scalar(p.dtype, p.beta)
    assert exact_case(p.dtype, al, be), p.name
    oracle.transform(p.dtype, p.op, p.alpha, p.beta, p.A, a_host.buffers(), p.B, b_host.buffers())
    n = count_mismatches(got_host.arena, a_host.arena)
    assert n == 0, f"{p.name}: {n} of {got_host.arena.size} elements differ from the oracle"


def blocks_have_no_nan(p, Ad):
    """A was pre-filled with NaN and beta = 0: every block element is written.
    For a layout whose buffers hold padding (a leading dimension above the
    local extent) the padding keeps its NaN, and the whole-buffer comparison
    with the oracle covers the blocks instead."""
    if p.A.numel() != int(np.sum(p.A.bufsize)):
        return True
    for r in range(p.A.nbuf):
        buf = Ad.buffer(r)
        covered = int(p.A.bufsize[r])
        assert covered == buf.numel()
        if torch.isnan(torch.view_as_real(buf) if buf.is_complex() else buf).any():
            return False
    return True


@pytest.mark.parametrize("name", ["c2", "c3", "c5", "c5b", "bc8", "ld1", "odd"])
def test_config_full_size(name, dev):
    import paper_2106_06601_gb300 as costa
    p = {**C.CONFIGS, **C.EXTRA_WORKLOADS}[name]()
    mat = Mat(p, dev)
    try:
        ij = sample_points(p.A, 200_000, 7)
        ia, ib = mat.sample_index(ij)
        a_pre = mat.Ad.arena[ia].cpu().numpy()
        b = mat.Bd.arena[ib].cpu().numpy()
        a_host, b_host = mat.Ad.download(), mat.Bd.download()
        b_bits = bits(mat.Bd.arena).clone()
        stream = torch.cuda.current_stream().cuda_stream
        sigma = costa.costa_transform(mat.LA, mat.LB, p.op, p.alpha, p.beta, relabel=True,
                                      stream=stream)
        torch.cuda.synchronize()
        a_post = mat.Ad.arena[ia].cpu().numpy()
        check_samples(p, a_pre, b, a_post)
        assert torch.equal(bits(mat.Bd.arena), b_bits), "B was modified"
        del b_bits
        if p.a_kind == "nan":
            assert blocks_have_no_nan(p, mat.Ad)
        whole_buffer_check(p, a_host, b_host, mat.Ad.download())
        del a_host, b_host
        V = costa.costa_volume(mat.LA, mat.LB, p.op, stream)
        assert V.sum() == p.A.m * p.A.n
        cf = json.load(open(GOLDEN)).get(name)
        best = oracle.lap_optimum(V)
        if cf:
            assert V.sum() == cf["total"] and best == cf["optimum"]
            assert set(np.unique(V).tolist()) == {0, cf["package"]}
        assert oracle.objective(V, sigma) == best
        st = costa.costa_plan_stats_get(mat.LA, mat.LB, p.op, relabel=True)
        assert st["local_relabeled"] == best
    finally:
        mat.close()


@pytest.mark.parametrize("name", ["zb", "za"])
def test_complex_scalars_full_size(name, dev):
    """c2's layouts with double complex data and complex scalars (zb: beta =
    0.5 + 0.25i, four products per component; za: alpha = 0.3 - 0.4i, beta =
    0, two), the kinds summed in fixed point on the integer pipes.  Every
    element of A is compared with the oracle, row slab by row slab, within
    2 ulp of the component's largest term; B must be bitwise unchanged."""
    import paper_2106_06601_gb300 as costa
    p = C.EXTRA_WORKLOADS[name]()
    mat = Mat(p, dev)
    try:
        a_host, b_host = mat.Ad.download(), mat.Bd.download()
        a_pre = a_host.arena.copy()
        b_bits = bits(mat.Bd.arena).clone()
        stream = torch.cuda.current_stream().cuda_stream
        costa.costa_transform(mat.LA, mat.LB, p.op, p.alpha, p.beta, relabel=True, stream=stream)
        torch.cuda.synchronize()
        assert torch.equal(bits(mat.Bd.arena), b_bits), "B was modified"
        del b_bits
        got = mat.Ad.download().arena
        oracle.transform(p.dtype, p.op, p.alpha, p.beta, p.A, a_host.buffers(), p.B, b_host.buffers())
        want = a_host.arena
        al, be = oracle.scalar(p.dtype, p.alpha), oracle.scalar(p.dtype, p.beta)
        assert not exact_case(p.dtype, al, be)
        rows = 256
        for i0 in range(0, p.A.m, rows):
            i1 = min(p.A.m, i0 + rows)
            ii, jj = np.meshgrid(np.arange(i0, i1), np.arange(p.A.n), indexing="ij")
            ij = np.stack([ii.ravel(), jj.ravel()], 1)
            _, abuf, aoff = oracle.locate(p.A, ij)
            _, bbuf, boff = oracle.locate(p.B, ij[:, ::-1].copy())
            ia, ib = a_host.starts[abuf] + aoff, b_host.starts[bbuf] + boff
            bvals = b_host.arena[ib].astype(np.complex128)
            if p.op == "C":
                bvals = np.conj(bvals)
            assert_close(p.dtype, got[ia], want[ia], al, be, bvals, a_pre[ia], exact=False)
        # padding and alignment gaps of A keep their values
        covered = np.zeros(got.size, bool)
        for i0 in range(0, p.A.m, 2048):
            ii, jj = np.meshgrid(np.arange(i0, min(p.A.m, i0 + 2048)), np.arange(p.A.n), indexing="ij")
            _, abuf, aoff = oracle.locate(p.A, np.stack([ii.ravel(), jj.ravel()], 1))
            covered[a_host.starts[abuf] + aoff] = True
        assert count_mismatches(got[~covered], a_pre[~covered]) == 0
    finally:
        mat.close()


def test_config_c3_volume_matches_oracle_count(dev):
    """c3's irregular target grid has no closed form: compare V with the
    oracle's element-by-element count."""
    import paper_2106_06601_gb300 as costa
    p = C.c3()
    mat = Mat(p, dev)
    try:
        V = costa.costa_volume(mat.LA, mat.LB, p.op, torch.cuda.current_stream().cuda_stream)
        assert np.array_equal(V, oracle.volume(p.op, p.A, p.B, 64))
    finally:
        mat.close()


def test_config_c4_batched(dev):
    import paper_2106_06601_gb300 as costa
    probs = C.c4()
    mats = [Mat(p, dev) for p in probs]
    try:
        idx = []
        for k, (p, m) in enumerate(zip(probs, mats)):
            ij = sample_points(p.A, 20_000, 100 + k)
            ia, ib = m.sample_index(ij)
            idx.append((ia, ib, m.Ad.arena[ia].cpu().numpy(), m.Bd.arena[ib].cpu().numpy()))
        hosts = [(m.Ad.download(), m.Bd.download()) for m in mats]
        b_bits = [bits(m.Bd.arena).clone() for m in mats]
        stream = torch.cuda.current_stream().cuda_stream
        sigma = costa.costa_transform_batched([m.LA for m in mats], [m.LB for m in mats],
                                              [p.op for p in probs], [p.alpha for p in probs],
                                              [p.beta for p in probs], relabel=True,
                                              stream=stream)
        torch.cuda.synchronize()
        for p, m, (ia, ib, a_pre, b) in zip(probs, mats, idx):
            check_samples(p, a_pre, b, m.Ad.arena[ia].cpu().numpy())
            assert blocks_have_no_nan(p, m.Ad)
        for p, m, bb, (a_host, b_host) in zip(probs, mats, b_bits, hosts):
            assert torch.equal(bits(m.Bd.arena), bb), f"{p.name}: B was modified"
            whole_buffer_check(p, a_host, b_host, m.Ad.download())
        st = costa.costa_plan_stats_get([m.LA for m in mats], [m.LB for m in mats],
                                        [p.op for p in probs], relabel=True)
        assert st["total_volume"] == 64 * 2048 * 3072
        assert sorted(sigma.tolist()) == list(range(16))
    finally:
        for m in mats:
            m.close()


def test_more_than_2_31_elements(dev):
    """A matrix of 65536 x 36864 f32 (2.4e9 elements, 9.7 GB per side): every
    element count, offset and volume sum passes 2^31.  Sampled outputs against
    the oracle; V sums to m * n; B bit-for-bit untouched."""
    import paper_2106_06601_gb300 as costa
    from workloads import layouts as L
    m, n = 65536, 36864
    perm = [(5 * k + 3) % 16 for k in range(16)]
    B = L.block_cyclic(m, n, 128, 128, 4, 4, name="B")
    A = L.block_cyclic(n, m, 256, 256, 4, 4, rank_perm=perm, name="A")
    p = C.Problem("big", "f32", "T", 2.0, 0.5, A, B, "uniform", "uniform", C.SEED0 + 31)
    assert p.A.m * p.A.n > 2 ** 31
    mat = Mat(p, dev)
    try:
        ij = sample_points(p.A, 100_000, 11)
        # the far corner, whose offsets are the largest
        ij = np.concatenate([ij, np.array([[p.A.m - 1, p.A.n - 1], [p.A.m - 1, 0], [0, p.A.n - 1]])])
        ia, ib = mat.sample_index(ij)
        a_pre = mat.Ad.arena[ia].cpu().numpy()
        b = mat.Bd.arena[ib].cpu().numpy()
        b_bits = bits(mat.Bd.arena).clone()
        stream = torch.cuda.current_stream().cuda_stream
        costa.costa_transform(mat.LA, mat.LB, p.op, p.alpha, p.beta, relabel=True, stream=stream)
        torch.cuda.synchronize()
        check_samples(p, a_pre, b, mat.Ad.arena[ia].cpu().numpy())
        assert torch.equal(bits(mat.Bd.arena), b_bits), "B was modified"
        del b_bits
        V = costa.costa_volume(mat.LA, mat.LB, p.op, stream)
        assert int(V.sum()) == p.A.m * p.A.n
    finally:
        mat.close()
        del mat
        torch.cuda.empty_cache()
