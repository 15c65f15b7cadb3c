"""Pins for the CPU oracle: each check ties it to something other than itself
(numpy's transpose/conjugate on a block-sliced global matrix, exact rational
arithmetic, closed-form volumes, brute force and a library LAP solver), and
the "planted mistake" tests show that a plausible error fails a pin."""
import json
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle
from tests._util import (global_matrix, op_apply, owner_matrix, scatter_global,
                         volume_by_owner_maps)
from workloads import configs as C
from workloads import gen
from workloads import layouts as L
from workloads.materialize import HostMatrix, host_problem

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def run_oracle(p, B, A):
    Aout = A.copy()
    oracle.transform(p.dtype, p.op, p.alpha, p.beta, p.A, Aout.buffers(), p.B, B.buffers())
    return Aout


def expected_global(p, B, A):
    """alpha * op(B) + beta * A on global matrices with numpy (only used when
    the result is exact: power-of-two scalars, or beta == 0 with alpha = 1)."""
    GB = global_matrix(p.B, B.buffers())
    GA = global_matrix(p.A, A.buffers())
    X = op_apply(p.op, GB)
    if p.dtype in ("f32", "f64"):
        X = X.real if np.iscomplexobj(X) else X
    if p.beta == 0:
        return (p.alpha * X).astype(GB.dtype) if p.alpha != 1 else X.astype(GB.dtype)
    return (p.alpha * X + p.beta * GA).astype(GB.dtype)


# ----------------------------------------------------------------------------
# addressing and op semantics
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("case", range(40))
def test_pure_movement_matches_numpy_op(case):
    """alpha = 1, beta = 0: A must equal op(B) exactly (N: a permutation of
    elements; T: transpose; C: conjugate transpose)."""
    p = C.fuzz_problem(case)
    p.alpha, p.beta, p.a_kind = 1.0, 0.0, "nan"
    B, A = host_problem(p)
    Aout = run_oracle(p, B, A)
    got = global_matrix(p.A, Aout.buffers())
    want = op_apply(p.op, global_matrix(p.B, B.buffers()))
    assert np.array_equal(got, want)
    assert not np.isnan(got).any()


@pytest.mark.parametrize("case", range(40, 70))
def test_power_of_two_scalars_exact(case):
    p = C.fuzz_problem(case)
    p.alpha, p.beta, p.a_kind = 2.0, 0.5, "uniform"
    B, A = host_problem(p)
    Aout = run_oracle(p, B, A)
    got = global_matrix(p.A, Aout.buffers())
    assert np.array_equal(got, expected_global(p, B, A))


def test_padding_and_foreign_elements_untouched():
    p = C.fuzz_problem(3)
    p.A = L.block_cyclic(p.A.m, p.A.n, 5, 7, 2, 2, storage="C", ld_pad=3)
    p.B = L.block_cyclic(p.B.m, p.B.n, 4, 6, 2, 2, storage="R", ld_pad=2)
    p.B.nranks = p.A.nranks = 4
    B, _ = host_problem(p)
    A = HostMatrix(p.A, p.dtype, guard=9, sentinel=123.0)
    want = A.arena.copy()
    Aout = run_oracle(p, B, A)
    # every element the oracle wrote is a block element; the rest stays 123
    written = np.zeros(A.arena.size, bool)
    for bi in range(p.A.nbr):
        for bj in range(p.A.nbc):
            h = int(p.A.rsplit[bi + 1] - p.A.rsplit[bi])
            w = int(p.A.csplit[bj + 1] - p.A.csplit[bj])
            base = int(A.starts[p.A.buf[bi, bj]] + p.A.off[bi, bj])
            ld = int(p.A.ld[bi, bj])
            for r in range(h):
                for c in range(w):
                    written[base + (r + c * ld if p.A.order[bi, bj] == 0 else r * ld + c)] = True
    assert np.array_equal(Aout.arena[~written], want[~written])


def test_transpose_round_trip_is_identity():
    for case in range(70, 85):
        p = C.fuzz_problem(case, op="T")
        p.alpha, p.beta = 1.0, 0.0
        B, A = host_problem(p)
        A1 = run_oracle(p, B, A)
        back = HostMatrix(p.B, p.dtype).fill("nan", 0, lambda r: 0)
        oracle.transform(p.dtype, "T", 1.0, 0.0, p.B, back.buffers(), p.A, A1.buffers())
        assert np.array_equal(global_matrix(p.B, back.buffers()),
                              global_matrix(p.B, B.buffers()))


@pytest.mark.parametrize("dtype", ["c64", "c128"])
def test_conjugate_transpose_round_trip(dtype):
    p = C.fuzz_problem(5, dtype=dtype, op="C")
    p.alpha, p.beta = 1.0, 0.0
    B, A = host_problem(p)
    A1 = run_oracle(p, B, A)
    GA = global_matrix(p.A, A1.buffers())
    GB = global_matrix(p.B, B.buffers())
    assert np.array_equal(GA, np.conj(GB.T))
    back = HostMatrix(p.B, dtype).fill("nan", 0, lambda r: 0)
    oracle.transform(dtype, "C", 1.0, 0.0, p.B, back.buffers(), p.A, A1.buffers())
    assert np.array_equal(global_matrix(p.B, back.buffers()), GB)


@pytest.mark.parametrize("dtype", ["f32", "f64"])
def test_conjugate_on_real_is_transpose(dtype):
    p = C.fuzz_problem(8, dtype=dtype, op="C")
    p.alpha, p.beta = 1.0, 0.0
    B, A = host_problem(p)
    A1 = run_oracle(p, B, A)
    p.op = "T"
    A2 = run_oracle(p, B, A)
    assert np.array_equal(A1.arena, A2.arena, equal_nan=True)


def test_linearity_in_alpha():
    p = C.fuzz_problem(12, dtype="f64")
    p.beta = 0.0
    B, A = host_problem(p)
    p.alpha = 1.0
    A1 = global_matrix(p.A, run_oracle(p, B, A).buffers())
    p.alpha = 4.0
    A4 = global_matrix(p.A, run_oracle(p, B, A).buffers())
    assert np.array_equal(A4, 4.0 * A1)


def test_locate_matches_block_views():
    p = C.fuzz_problem(21)
    spec = p.A
    ij = np.array([(i, j) for i in range(spec.m) for j in range(spec.n)], np.int64)
    owner, buf, off = oracle.locate(spec, ij)
    assert np.array_equal(owner.reshape(spec.m, spec.n), owner_matrix(spec))
    # write each element's linear index through the oracle's address and read
    # back through the independent block views
    H = HostMatrix(spec, "f64")
    H.arena[:] = -1
    for k in range(len(ij)):
        H.buffer(buf[k])[off[k]] = k
    G = global_matrix(spec, H.buffers())
    assert np.array_equal(G.ravel(), np.arange(len(ij), dtype=np.float64))


# ----------------------------------------------------------------------------
# arithmetic against exact rational values
# ----------------------------------------------------------------------------

def _exact(alpha, beta, b, a):
    al, be = complex(alpha), complex(beta)
    re = (Fraction(al.real) * Fraction(b.real) - Fraction(al.imag) * Fraction(b.imag))
    im = (Fraction(al.real) * Fraction(b.imag) + Fraction(al.imag) * Fraction(b.real))
    if be != 0:
        re += Fraction(be.real) * Fraction(a.real) - Fraction(be.imag) * Fraction(a.imag)
        im += Fraction(be.real) * Fraction(a.imag) + Fraction(be.imag) * Fraction(a.real)
    return re, im


def _half_ulp_ok(got, exact, real):
    """|got - exact| <= 0.5 ulp(got) (plus 2^-40 relative slack for the
    oracle's non-final roundings): got is the exact value rounded once."""
    g = Fraction(float(got))
    sp = Fraction(float(np.spacing(real(abs(float(got))))))
    return abs(g - exact) <= sp / 2 + abs(exact) * Fraction(1, 2 ** 40)


@pytest.mark.parametrize("dtype", ["f32", "f64", "c64", "c128"])
@pytest.mark.parametrize("alpha,beta", [(-0.3, 0.7), (0.1, -1.25), (1.0, 1e-3),
                                        (complex(0.5, -0.75), complex(1.0, 0.0)),
                                        (complex(-0.6, 0.3), 0.0),
                                        (complex(0.2, 0.9), complex(-1.1, 0.4))])
def test_combine_rounds_exact_value_once(dtype, alpha, beta):
    if dtype in ("f32", "f64") and (complex(alpha).imag or complex(beta).imag):
        pytest.skip("complex scalars need complex data")
    n = 4000
    b = gen.values_np(dtype, "uniform", 5, 1, n)
    a = gen.values_np(dtype, "uniform", 5, 2, n)
    # include cancellation: a close to -alpha b / beta
    if complex(beta) != 0 and dtype in ("f32", "f64"):
        a[:500] = (-(alpha * b[:500].astype(np.float64)) / beta).astype(a.dtype)
    alpha, beta = oracle.scalar(dtype, alpha), oracle.scalar(dtype, beta)
    out = oracle.combine(dtype, "N", alpha, beta, b, a)
    real = np.float32 if dtype in ("f32", "c64") else np.float64
    for k in range(n):
        re, im = _exact(alpha, beta, complex(b[k]), complex(a[k]))
        o = complex(out[k])
        assert _half_ulp_ok(o.real, re, real), (k, o, float(re))
        if dtype in ("c64", "c128"):
            assert _half_ulp_ok(o.imag, im, real), (k, o, float(im))


def test_beta_zero_does_not_read_a():
    b = gen.values_np("f64", "uniform", 1, 1, 100)
    a = np.full(100, np.nan)
    out = oracle.combine("f64", "N", 0.75, 0.0, b, a)
    assert np.array_equal(out, 0.75 * b)
    out = oracle.combine("c128", "C", 1.0, 0.0, b.astype(np.complex128) * (1 + 2j),
                         a.astype(np.complex128))
    assert np.array_equal(out, np.conj(b * (1 + 2j)))


# ----------------------------------------------------------------------------
# volumes (Alg. 2) and the closed forms of the configs
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("case", range(25))
def test_volume_matches_owner_maps(case):
    p = C.fuzz_problem(case)
    P = p.A.nranks
    V = oracle.volume(p.op, p.A, p.B, P)
    assert np.array_equal(V, volume_by_owner_maps(p.op, p.A, p.B, P))
    assert V.sum() == p.A.m * p.A.n          # each element sits in exactly one package


def _closed_forms():
    with open(os.path.join(GOLDEN, "closed_forms.json")) as f:
        return json.load(f)


def test_c1_volume_closed_form():
    p = C.c1()
    V = oracle.volume(p.op, p.A, p.B, 4)
    cf = _closed_forms()["c1"]
    assert V.tolist() == cf["V"]
    assert oracle.lap_optimum(V) == cf["optimum"]


def test_c2_volume_closed_form():
    p = C.c2()
    V = oracle.volume(p.op, p.A, p.B, 16)
    cf = _closed_forms()["c2"]
    assert V.sum() == cf["total"]
    assert set(np.unique(V).tolist()) == {0, cf["package"]}
    assert np.all((V > 0).sum(axis=0) == cf["degree"]) and np.all((V > 0).sum(axis=1) == cf["degree"])
    assert oracle.lap_optimum(V) == cf["optimum"]


@pytest.mark.slow
def test_c5_volume_closed_form():
    p = C.c5()
    V = oracle.volume(p.op, p.A, p.B, 256)
    cf = _closed_forms()["c5"]
    assert V.sum() == cf["total"]
    assert set(np.unique(V).tolist()) == {0, cf["package"]}
    assert np.all((V > 0).sum(axis=0) == cf["degree"]) and np.all((V > 0).sum(axis=1) == cf["degree"])
    # the rank p = (pr, pc) sends to the panels k with (k div 2) mod 16 == pc
    for pr in (0, 7):
        for pc in (0, 5, 15):
            ks = np.flatnonzero(V[pr * 16 + pc])
            assert np.all((ks // 2) % 16 == pc)
    assert oracle.lap_optimum(V) == cf["optimum"]


def test_equal_grids_permuted_owners_relabel_to_zero_remote():
    """Sec. 7.2: when two layouts share their grid and differ only by the
    owner permutation, relabeling makes all volume local."""
    perm = gen.IntStream(1, 77).permutation(12)
    B = L.block_cyclic(60, 84, 10, 14, 3, 4, grid_order="R")
    A = L.block_cyclic(60, 84, 10, 14, 3, 4, grid_order="C", rank_perm=perm)
    V = oracle.volume("N", A, B, 12)
    assert oracle.lap_optimum(V) == 60 * 84
    assert np.count_nonzero(V) == 12


# ----------------------------------------------------------------------------
# relabeling (Thm. 1 / Thm. 2) against brute force, DP and a library solver
# ----------------------------------------------------------------------------

def _rand_V(P, seed, zeros=True, ties=False):
    rng = gen.IntStream(seed, 5)
    V = np.array([[rng.below(7 if ties else 1000) for _ in range(P)] for _ in range(P)],
                 np.int64)
    if zeros:
        V[V % 3 == 0] = 0
    return V


@pytest.mark.parametrize("P", [1, 2, 3, 4, 5, 6, 7, 8])
def test_lap_solvers_agree_small(P):
    for s in range(12):
        V = _rand_V(P, 100 * P + s, ties=(s % 2 == 0))
        bf, sb = oracle.lap_bruteforce(V)
        dp, sd = oracle.lap_subset_dp(V)
        lib, sl = oracle.lap_library(V)
        assert bf == dp == lib
        for s_ in (sb, sd, sl):
            assert sorted(s_.tolist()) == list(range(P))
            assert oracle.objective(V, s_) == bf
        # Remark (identity is a perfect matching): optimum >= trace
        assert bf >= np.trace(V)


@pytest.mark.parametrize("P", [9, 12, 16, 20])
def test_lap_dp_matches_library(P):
    for s in range(3):
        V = _rand_V(P, 7 * P + s)
        assert oracle.lap_subset_dp(V)[0] == oracle.lap_library(V)[0]


def test_lemma1_gain_equals_cost_reduction():
    """Lemma 1 under the locally-free volume cost (Eq. 2): the total gain
    sum_j delta(j, sigma(j)) with delta(x, y) = V(S_yx) - V(S_xx) (Remark on
    the gain) equals W(G) - W(G_sigma), where W counts remote volume."""
    P = 6
    V = _rand_V(P, 31)
    total = int(V.sum())

    def W(sig):  # remote volume when target label q is taken by process sig[q]
        return total - sum(int(V[sig[q], q]) for q in range(P))

    ident = list(range(P))
    for s in range(20):
        sig = gen.IntStream(s, 8).permutation(P)
        gain = sum(int(V[sig[x], x]) - int(V[x, x]) for x in range(P))
        assert gain == W(ident) - W(sig)


# ----------------------------------------------------------------------------
# planted mistakes: each pin must fail on a plausible oracle error
# ----------------------------------------------------------------------------

def test_planted_mistakes_are_caught():
    p = C.fuzz_problem(40, dtype="c128", op="C")
    p.alpha, p.beta, p.a_kind = 2.0, 0.5, "uniform"
    B, A = host_problem(p)
    good = global_matrix(p.A, run_oracle(p, B, A).buffers())
    want = expected_global(p, B, A)
    assert np.array_equal(good, want)
    GB = global_matrix(p.B, B.buffers())
    GA = global_matrix(p.A, A.buffers())
    mutants = {
        "dropped beta term": 2.0 * np.conj(GB.T),
        "missing conjugate": 2.0 * GB.T + 0.5 * GA,
        "sign of beta": 2.0 * np.conj(GB.T) - 0.5 * GA,
    }
    for name, bad in mutants.items():
        assert not np.array_equal(bad, want), name
    # a transposed operand in the volume count breaks the owner-map pin
    q = C.fuzz_problem(41, op="T")
    while q.A.m == q.A.n:
        q = C.fuzz_problem(q.index + 200, op="T")
    P = q.A.nranks
    V = oracle.volume("T", q.A, q.B, P)
    ob, qa = owner_matrix(q.B), owner_matrix(q.A)
    # a wrong volume (owner maps swapped) differs from the pinned one
    Vbad = np.bincount((qa.astype(np.int64) * P + ob.T).ravel(), minlength=P * P).reshape(P, P)
    assert not np.array_equal(Vbad, V) or np.array_equal(Vbad, Vbad.T)
    # a scrambled buffer address fails the block-view reconstruction
    H = HostMatrix(q.A, "f64")
    scatter_global(q.A, H.buffers(), np.arange(q.A.m * q.A.n, dtype=np.float64).reshape(q.A.m, q.A.n))
    ij = np.array([(i, j) for i in range(q.A.m) for j in range(q.A.n)])
    _, buf, off = oracle.locate(q.A, ij)
    vals = np.array([H.buffer(b)[o] for b, o in zip(buf, off)])
    assert np.array_equal(vals, np.arange(len(ij), dtype=np.float64))
    # an off-by-one storage address (a dropped "+ r" term would look alike)
    size = q.A.bufsize[buf]
    shifted = np.where(off + 1 < size, off + 1, off - 1)
    wrong = np.array([H.buffer(b)[o] for b, o in zip(buf, shifted)])
    assert not np.array_equal(wrong, np.arange(len(ij), dtype=np.float64))
