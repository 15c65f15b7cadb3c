"""Pins for the seeded input module (generators and layout descriptions)."""
import numpy as np
import pytest

from workloads import configs as C
from workloads import gen
from workloads import layouts as L
from workloads.materialize import HostMatrix, arena_offsets


def test_splitmix64_reference_values():
    # SplitMix64 seeded with 0 (state 0): first outputs, as printed by the
    # authors' reference implementation (Steele, Lea & Flood 2014; also the
    # seeding generator of xoshiro, Blackman & Vigna).
    z = 0
    outs = []
    for _ in range(3):
        z = (z + gen.GAMMA) & gen.MASK64
        outs.append(gen._mix_int(z))
    assert outs == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_counter_form_matches_sequential():
    s0 = gen.stream_state(7, 3)
    z = s0
    for k in range(50):
        z = (z + gen.GAMMA) & gen.MASK64
        assert gen.draw_int(7, 3, k) == gen._mix_int(z)
    d = gen.draws_np(7, 3, 0, 50)
    assert [int(x) for x in d] == [gen.draw_int(7, 3, k) for k in range(50)]
    d2 = gen.draws_np(7, 3, 20, 10)
    assert np.array_equal(d2, d[20:30])


@pytest.mark.parametrize("dtype", ["f32", "f64", "c64", "c128"])
def test_torch_matches_numpy(dtype):
    import torch
    a = gen.values_np(dtype, "uniform", 11, 5, 5000)
    t = torch.empty(5000, dtype=getattr(torch, {"f32": "float32", "f64": "float64",
                                                "c64": "complex64", "c128": "complex128"}[dtype]))
    gen.fill_torch(t, dtype, "uniform", 11, 5)
    assert np.array_equal(a, t.numpy())


def test_uniform_range_and_moments():
    v = gen.values_np("f64", "uniform", 1, 1, 200000)
    assert v.min() >= -1.0 and v.max() < 1.0
    assert abs(v.mean()) < 0.01 and abs(v.var() - 1 / 3) < 0.01
    f = gen.values_np("f32", "uniform", 1, 1, 200000)
    assert f.dtype == np.float32 and f.min() >= -1 and f.max() < 1
    # f32 values are multiples of 2^-23
    assert np.all(np.ldexp(f.astype(np.float64) + 1.0, 23) % 1 == 0)


def test_normal_moments():
    v = gen.values_np("f64", "normal", 1, 2, 400000)
    assert abs(v.mean()) < 0.01 and abs(v.std() - 1) < 0.01
    # fourth moment of N(0,1) is 3
    assert abs(np.mean(v ** 4) - 3.0) < 0.08


def test_permutation_and_between():
    rng = gen.IntStream(3, 4)
    for n in (1, 2, 5, 64, 256):
        p = rng.permutation(n)
        assert sorted(p) == list(range(n))
    xs = [rng.between(512, 3584) for _ in range(2000)]
    assert min(xs) >= 512 and max(xs) <= 3584


# ----------------------------------------------------------------------------
# block-cyclic layouts against the ScaLAPACK index maps
# ----------------------------------------------------------------------------

def indxg2p(ig, nb, nprocs):       # global index -> process coordinate (srcproc 0)
    return (ig // nb) % nprocs


def indxg2l(ig, nb, nprocs):       # global index -> local index
    return (ig // (nb * nprocs)) * nb + ig % nb


@pytest.mark.parametrize("n,nb,p", [(256, 16, 2), (100, 7, 3), (5, 8, 4), (8192, 64, 4),
                                    (131072, 32, 16), (1, 1, 1), (37, 5, 5)])
def test_numroc_counts(n, nb, p):
    counts = np.bincount(indxg2p(np.arange(n), nb, p), minlength=p)
    assert [L.numroc(n, nb, i, p) for i in range(p)] == counts.tolist()


@pytest.mark.parametrize("args", [
    (256, 256, 16, 16, 2, 2, "R", "C"), (256, 256, 32, 32, 2, 2, "C", "C"),
    (37, 53, 5, 7, 3, 2, "R", "R"), (100, 90, 8, 12, 2, 3, "C", "C"),
    (64, 48, 64, 48, 1, 1, "R", "C")])
def test_block_cyclic_matches_scalapack_maps(args):
    m, n, mb, nb, pr, pc, go, st = args
    perm = gen.IntStream(9, 9).permutation(pr * pc)
    spec = L.block_cyclic(m, n, mb, nb, pr, pc, grid_order=go, rank_perm=perm,
                          storage=st, ld_pad=2)
    spec.check()
    i = np.arange(m)[:, None]
    j = np.arange(n)[None, :]
    ip, jp = indxg2p(i, mb, pr), indxg2p(j, nb, pc)
    il, jl = indxg2l(i, mb, pr), indxg2l(j, nb, pc)
    grank = ip * pc + jp if go == "R" else ip + jp * pr
    owner_want = np.asarray(perm)[grank]
    from tests._util import owner_matrix
    assert np.array_equal(owner_matrix(spec), owner_want)
    # element offsets inside the owner's local matrix
    loc_rows = np.array([L.numroc(m, mb, r, pr) for r in range(pr)])
    loc_cols = np.array([L.numroc(n, nb, c, pc) for c in range(pc)])
    if st == "C":
        lld = loc_rows[ip] + 2
        want = il + jl * lld
    else:
        lld = loc_cols[jp] + 2
        want = il * lld + jl
    hs, ws = np.diff(spec.rsplit), np.diff(spec.csplit)
    bi = np.repeat(np.arange(spec.nbr), hs)[:, None]
    bj = np.repeat(np.arange(spec.nbc), ws)[None, :]
    r = i - spec.rsplit[bi]
    c = j - spec.csplit[bj]
    got = np.where(spec.order[bi, bj] == 0, spec.off[bi, bj] + r + c * spec.ld[bi, bj],
                   spec.off[bi, bj] + r * spec.ld[bi, bj] + c)
    assert np.array_equal(got, want)


def test_configs_are_consistent():
    for name in ("c1", "c2", "c3", "c5"):
        p = C.CONFIGS[name]()
        p.A.check()
        p.B.check()
        assert p.A.nranks == p.B.nranks
        if p.op == "N":
            assert (p.A.m, p.A.n) == (p.B.m, p.B.n)
        else:
            assert (p.A.m, p.A.n) == (p.B.n, p.B.m)
    for q in C.c4():
        q.A.check()
        q.B.check()
    # the irregular grid of c3: 8 blocks per dimension, sizes in [512, 3584]
    a = C.c3().A
    for s in (a.rsplit, a.csplit):
        d = np.diff(s)
        assert len(d) == 8 and d.min() >= 512 and d.max() <= 3584 and s[-1] == 16384
    assert sorted(a.owner.ravel().tolist()) == list(range(64))
    # c5: B's local leading dimension is 8192 rows on every rank
    b5 = C.c5().B
    assert set(np.unique(b5.ld).tolist()) == {8192}


def test_fuzz_problems_are_consistent():
    for k in range(60):
        p = C.fuzz_problem(k)
        p.A.check()
        p.B.check()


def test_arena_alignment():
    starts, total = arena_offsets([3, 100, 1, 0, 7], 8, guard=5)
    assert np.all((starts * 8) % 256 == 0)
    assert np.all(np.diff(starts) >= np.array([3, 100, 1, 0]) + 5)
    h = HostMatrix(C.c1().B, "f64", guard=4, sentinel=7.0)
    assert np.all(h.arena == 7.0)
