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


@pytest.mark.parametrize("case", [21, 8, 30])
def test_locate_matches_block_views(case):
    """Cases 8 and 30 have an empty block row or column."""
    p = C.fuzz_problem(case)
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
# cost function, COPR and greedy against hand-worked cases (tests/golden)
# ----------------------------------------------------------------------------

def _relabel_cases():
    with open(os.path.join(GOLDEN, "relabel_cases.json")) as f:
        return json.load(f)


def test_cost_W_topology_3x3_by_hand():
    """W(G_sigma) of every permutation, the COPR optimum (Def. COPR) and the
    volume-only optimum (Eq. 2) of the hand-worked 3 x 3 case."""
    g = _relabel_cases()["topology_3x3"]
    V, lat, bw = np.array(g["V"]), np.array(g["lat"], float), np.array(g["bw"], float)
    for key, w in g["W"].items():
        sigma = [int(x) for x in key.split(",")]
        assert oracle.cost_W(V, lat, bw, sigma) == w, key
        assert oracle.objective(V, sigma) == g["local"][key], key
    best, sigma = oracle.copr_bruteforce_cost(V, lat, bw)
    assert best == g["optimum"] and sigma.tolist() == g["sigma"]
    vbest, vsig = oracle.lap_bruteforce(V)
    assert vbest == g["volume_optimum"] and vsig.tolist() == g["volume_sigma"]


def test_cost_W_closed_forms():
    """W(G_sigma) on cases whose totals are derived by hand (golden README)."""
    g = _relabel_cases()["cost_W_closed_forms"]
    f = g["all_ones_identity"]
    for P, want in zip(f["P"], f["values"]):
        idx = np.arange(P)
        V = np.ones((P, P), np.int64)
        lat = 1.0 - np.eye(P)
        bw = np.abs(idx[:, None] - idx[None, :]).astype(float)
        assert oracle.cost_W(V, lat, bw, idx) == want == P * (P - 1) + (P ** 3 - P) // 3
    P = 4
    idx = np.arange(P)
    V = np.tile(1 + idx, (P, 1)).astype(np.int64)     # V[i][j] = 1 + j
    lat = 1.0 - np.eye(P)
    bw = np.abs(idx[:, None] - idx[None, :]).astype(float)
    assert oracle.cost_W(V, lat, bw, (idx + 1) % P) == g["shift_4"]["W"]
    d = g["diagonal_nonzero"]
    P = d["P"]
    ones = np.ones((P, P))
    assert oracle.cost_W(np.ones((P, P), np.int64), ones, ones, np.arange(P)) == d["W"] \
        == 2 * P * (P - 1)


def test_greedy_hand_worked_with_ties():
    """Sec. 6 greedy: decreasing volume, ties by smaller p then smaller q."""
    g = _relabel_cases()["greedy_ties_4x4"]
    V = np.array(g["V"], np.int64)
    total, sigma = oracle.lap_greedy(V)
    assert sigma.tolist() == g["greedy_sigma"] and total == g["greedy_local"]
    assert oracle.lap_bruteforce(V)[0] == g["optimum"]


@pytest.mark.parametrize("P", [1, 2, 3, 4, 5, 6, 7])
def test_copr_reduces_to_volume_relabeling(P):
    """lat = 0, bw = 1 off the diagonal is the locally-free volume cost
    (Eq. 2): min W(G_sigma) = total volume - the volume optimum, and the
    minimizing sigma keeps that optimum (Remark on the gain)."""
    for s in range(6):
        V = _rand_V(P, 900 + 10 * P + s, ties=(s % 2 == 0))
        lat = np.zeros((P, P))
        bw = 1.0 - np.eye(P)
        best, sigma = oracle.copr_bruteforce_cost(V, lat, bw)
        opt, _ = oracle.lap_bruteforce(V)
        assert best == V.sum() - opt
        assert oracle.objective(V, sigma) == opt


@pytest.mark.parametrize("P", [2, 3, 5, 7])
def test_copr_latency_only_counts_remote_packages(P):
    """lat = 1 off the diagonal, bw = 0: W counts the remote non-empty
    packages, so min W = (non-empty packages) - (largest matching inside
    the support of V), the matching taken by brute force on V > 0."""
    for s in range(6):
        V = _rand_V(P, 700 + 10 * P + s)
        lat = 1.0 - np.eye(P)
        bw = np.zeros((P, P))
        best, _ = oracle.copr_bruteforce_cost(V, lat, bw)
        match, _ = oracle.lap_bruteforce((V > 0).astype(np.int64))
        assert best == np.count_nonzero(V) - match


# ----------------------------------------------------------------------------
# planted mistakes: mutated builds of the oracle itself must fail the pins
# ----------------------------------------------------------------------------

# (name, text in costa_oracle.c, replacement, replace every occurrence)
MUTANTS = [
    ("dropped beta term", "{alpha[0], beta[0]}, y[2] = {b[0], a[0]}",
     "{alpha[0], 0.0}, y[2] = {b[0], a[0]}", False),
    ("sign of beta", "{alpha[0], beta[0]}, y[2] = {b[0], a[0]}",
     "{alpha[0], -beta[0]}, y[2] = {b[0], a[0]}", False),
    ("missing conjugate", "Bbufs[bb], ob, b);\n            if (op == O_C && cplx) b[1] = -b[1];",
     "Bbufs[bb], ob, b);", False),
    ("sign of alpha's imaginary part", "double xr[4] = {alpha[0], -alpha[1], beta[0], -beta[1]};",
     "double xr[4] = {alpha[0], alpha[1], beta[0], -beta[1]};", False),
    ("product error term dropped", "*e = fma(a, b, -x);", "*e = 0.0;", False),
    ("beta = 0 reads A", "int beta0 = (beta[0] == 0.0 && beta[1] == 0.0);", "int beta0 = 0;", True),
    ("off-by-one row offset", "int64_t r = i - L->rsplit[bi], c = j - L->csplit[bj];",
     "int64_t r = i - L->rsplit[bi] + 1, c = j - L->csplit[bj];", False),
    ("storage orders swapped", "(L->order[b] == 0 ? r + c * L->ld[b] : r * L->ld[b] + c)",
     "(L->order[b] == 1 ? r + c * L->ld[b] : r * L->ld[b] + c)", False),
    ("column block from the row index", "int64_t bj = find_block(L->csplit, L->nbc, j);",
     "int64_t bj = find_block(L->csplit, L->nbc, i);", False),
    ("volume indices transposed", "loc[(int64_t)qb * P + qa] += 1;", "loc[(int64_t)qa * P + qb] += 1;",
     False),
    ("op ignored in volume", "else oracle_locate(B, j, i, &qb, &bb, &ob);\n                loc",
     "else oracle_locate(B, i, j, &qb, &bb, &ob);\n                loc", False),
    ("brute force minimizes", "if (s > best) {", "if (s < best || best == INT64_MIN) {", False),
    ("subset DP operand transposed", "best[S & ~((size_t)1 << p)] + V[(int64_t)p * P + q];",
     "best[S & ~((size_t)1 << p)] + V[(int64_t)q * P + p];", False),
    ("greedy tie rule reversed", "(V[key] == V[a] && key < a)", "(V[key] == V[a] && key > a)", False),
    ("greedy ascending", "int before = V[key] > V[a] ||", "int before = V[key] < V[a] ||", False),
    ("cost without latency", "W += lat[(int64_t)i * P + k] + bw", "W += bw", False),
    ("cost indexed by label", "W += lat[(int64_t)i * P + k] + bw[(int64_t)i * P + k] * (double)v;",
     "W += lat[(int64_t)i * P + j] + bw[(int64_t)i * P + j] * (double)v;", False),
    ("empty packages charged", "if (v == 0) continue;\n            int k = sigma[j];",
     "int k = sigma[j];", False),
    ("kept packages charged", "if (k == i) continue;\n            W +=", "W +=", False),
    ("COPR maximizes", "if (first || W < best) {", "if (first || W > best) {", False),
]


def _pins_for(name):
    """The pins that must catch each mutant (plain calls of the pin tests)."""
    cases_movement = lambda: [test_pure_movement_matches_numpy_op(c) for c in range(8)]
    cases_pow2 = lambda: [test_power_of_two_scalars_exact(c) for c in range(40, 52)]
    return {
        "dropped beta term": cases_pow2,
        "sign of beta": cases_pow2,
        "missing conjugate": lambda: test_conjugate_transpose_round_trip("c128"),
        "sign of alpha's imaginary part":
            lambda: test_combine_rounds_exact_value_once("c128", complex(0.2, 0.9), complex(-1.1, 0.4)),
        "product error term dropped": lambda: test_combine_rounds_exact_value_once("f64", -0.3, 0.7),
        "beta = 0 reads A": cases_movement,
        "off-by-one row offset": lambda: test_locate_matches_block_views(21),
        "storage orders swapped": lambda: test_locate_matches_block_views(21),
        "column block from the row index": lambda: [test_locate_matches_block_views(c) for c in (21, 8, 30)],
        "volume indices transposed": lambda: [test_volume_matches_owner_maps(c) for c in range(10)],
        "op ignored in volume": lambda: [test_volume_matches_owner_maps(c) for c in range(10)],
        "brute force minimizes": lambda: test_lap_solvers_agree_small(4),
        "subset DP operand transposed": lambda: test_lap_solvers_agree_small(5),
        "greedy tie rule reversed": test_greedy_hand_worked_with_ties,
        "greedy ascending": test_greedy_hand_worked_with_ties,
        "cost without latency": test_cost_W_closed_forms,
        "cost indexed by label": test_cost_W_closed_forms,
        "empty packages charged": test_cost_W_topology_3x3_by_hand,
        "kept packages charged": test_cost_W_closed_forms,
        "COPR maximizes": lambda: test_copr_reduces_to_volume_relabeling(4),
    }[name]


@pytest.fixture(scope="module")
def mutant_libs(tmp_path_factory):
    from concurrent.futures import ThreadPoolExecutor
    src = oracle.source_text()
    d = tmp_path_factory.mktemp("oracle_mutants")
    jobs = {}
    for k, (name, old, new, every) in enumerate(MUTANTS):
        n = src.count(old)
        assert n >= 1 and (every or n == 1), (name, n)
        jobs[name] = (src.replace(old, new), str(d / f"mutant{k}.so"))
    with ThreadPoolExecutor(8) as ex:
        futs = {name: ex.submit(oracle.compile_variant, text, path)
                for name, (text, path) in jobs.items()}
        return {name: f.result() for name, f in futs.items()}


@pytest.mark.parametrize("name", [m[0] for m in MUTANTS])
def test_planted_mistake_fails_a_pin(name, mutant_libs):
    pin = _pins_for(name)
    pin()                                   # the pin holds for the real oracle
    with oracle.loaded(mutant_libs[name]):
        try:
            pin()
        except Exception:
            return
    raise AssertionError(f"planted mistake '{name}' passed its pins")
