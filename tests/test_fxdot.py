"""The fixed-point sum of products that the kernels use for complex scalars
on double complex data (Eq. 1 with complex alpha or beta), run on the host
through costa_debug_fxdot, which compiles the kernels' own code.

Pinned against exact rational arithmetic (fractions.Fraction), against
hand-worked closed forms (exact sums, a round-to-even tie, total
cancellation), and against the oracle's component of alpha * b + beta * a.
The bound is the one the GPU parity tests assert, 2 ulp of the largest term,
and the evaluation's own claim is tighter: 0.5 ulp of the result plus
n * 2^-7 ulp of the largest product."""
import math
import random
from fractions import Fraction

import numpy as np
import pytest

import oracle
import paper_2106_06601_gb300 as costa


def _draw(rng):
    k = rng.random()
    if k < 0.05:
        return 0.0
    if k < 0.10:
        return rng.choice([1.0, -1.0, 0.5, 2.0 ** -480, -(2.0 ** 479) * 1.999, 2.0 ** 479 * 1.9999999])
    sign = rng.choice([-1.0, 1.0])
    if k < 0.80:
        return sign * rng.uniform(0.5, 1) * 2.0 ** rng.randint(-60, 60)
    return sign * rng.uniform(0.5, 1) * 2.0 ** rng.randint(-470, 470)


def _cases(n, count, seed):
    rng = random.Random(seed)
    x = np.empty((count, n))
    y = np.empty((count, n))
    neg = np.empty((count, n), np.int32)
    for k in range(count):
        for i in range(n):
            x[k, i], y[k, i], neg[k, i] = _draw(rng), _draw(rng), rng.randint(0, 1)
        if n == 4 and rng.random() < 0.4:  # term 2 cancels term 0 to a few bits
            y2 = y[k, 0] * (1 + rng.choice([0.0, 2.0 ** -52, -(2.0 ** -52), 2.0 ** -30]))
            if y2 == 0 or 2.0 ** -480 <= abs(y2) < 2.0 ** 480:
                x[k, 2], y[k, 2], neg[k, 2] = x[k, 0], y2, 1 - neg[k, 0]
    return x, y, neg


@pytest.mark.parametrize("n", [2, 4])
def test_fxdot_within_its_bound_of_the_exact_sum(n):
    x, y, neg = _cases(n, 20000, 11 + n)
    got = costa.costa_debug_fxdot(x, y, neg)
    for k in range(x.shape[0]):
        prods = [Fraction(x[k, i]) * Fraction(y[k, i]) * (-1 if neg[k, i] else 1) for i in range(n)]
        exact = sum(prods)
        M = max(abs(p) for p in prods)
        if M == 0:
            assert got[k] == 0.0
            continue
        ulp_m = Fraction(math.ulp(float(M)))
        rounded = float(exact)
        bound = Fraction(math.ulp(rounded)) / 2 + n * ulp_m / 128 if rounded else n * ulp_m / 128
        assert abs(Fraction(float(got[k])) - exact) <= bound, (k, x[k], y[k], neg[k], got[k], rounded)


def test_fxdot_closed_forms():
    t = 2.0 ** -27
    cases = [
        # (x, y, neg, expected)
        ([1.0, 1.0], [1.0, 1.0], [0, 0], 2.0),                        # exact sum
        ([3.0, 5.0], [7.0, 11.0], [0, 1], 21.0 - 55.0),               # exact, negative
        ([1.5, 1.5], [2.0 ** 100, 2.0 ** 100], [0, 1], 0.0),           # total cancellation gives +0
        ([1.0, t], [1.0, 2 * t], [0, 0], 1.0),                        # 1 + 2^-53: tie, to even (1)
        ([1.0, t], [1.0 + 2.0 ** -52, 2 * t], [0, 0], 1.0 + 2.0 ** -51),  # tie, to even (up)
        ([0.1, 0.2, 0.3, 0.4], [1.0, 1.0, 1.0, 1.0], [0, 0, 0, 0],
         float(Fraction(0.1) + Fraction(0.2) + Fraction(0.3) + Fraction(0.4))),
        ([2.0 ** 479 * 1.5, 2.0 ** 479 * 1.5], [2.0 ** 479, 2.0 ** 479], [0, 0], 1.5 * 2.0 ** 959),
        ([2.0 ** -480, 0.0], [2.0 ** -480, 5.0], [1, 0], -(2.0 ** -960)),  # smallest product
    ]
    for x, y, neg, want in cases:
        got = costa.costa_debug_fxdot(np.array([x]), np.array([y]), np.array([neg]))[0]
        assert got == want and math.copysign(1, got) == math.copysign(1, want), (x, y, neg, got, want)


@pytest.mark.parametrize("bad", [5e-324, 2.0 ** -481, 2.0 ** 480, float("inf"), float("nan")])
def test_fxdot_rejects_factors_outside_its_range(bad):
    with pytest.raises(costa.CostaError) as e:
        costa.costa_debug_fxdot(np.array([[1.0, bad]]), np.array([[1.0, 1.0]]), np.array([[0, 0]]))
    assert e.value.status == 1


@pytest.mark.parametrize("alpha,beta", [(complex(0.3, -0.4), 0.0), (1.0, complex(0.5, 0.25)),
                                        (complex(-1.1, 0.4), complex(0.2, 0.9))])
def test_fxdot_agrees_with_the_oracle_combine(alpha, beta):
    """The oracle's c128 component of alpha * b + beta * a (Dot2) against the
    kernels' fixed-point evaluation of the same products, within the GPU
    tests' 2 ulp(M); a third of the elements are set up so that the real
    part's products cancel."""
    rng = np.random.default_rng(5)
    count = 20000
    b = rng.uniform(-1, 1, count) + 1j * rng.uniform(-1, 1, count)
    a = rng.uniform(-1, 1, count) + 1j * rng.uniform(-1, 1, count)
    al, be = complex(alpha), complex(beta)
    if be != 0:
        third = count // 3
        # beta_r a_r = -(alpha_r b_r - alpha_i b_i) to within rounding
        a.real[:third] = -(al.real * b.real[:third] - al.imag * b.imag[:third]) / be.real
    want = oracle.combine("c128", "N", alpha, beta, b, a)
    re_x = np.stack([np.full(count, al.real), np.full(count, al.imag),
                     np.full(count, be.real), np.full(count, be.imag)], 1)
    re_y = np.stack([b.real, b.imag, a.real, a.imag], 1)
    re_n = np.tile(np.array([0, 1, 0, 1], np.int32), (count, 1))
    im_x = re_x
    im_y = np.stack([b.imag, b.real, a.imag, a.real], 1)
    im_n = np.zeros((count, 4), np.int32)
    got = (costa.costa_debug_fxdot(re_x, re_y, re_n) + 1j * costa.costa_debug_fxdot(im_x, im_y, im_n))
    from tests._util import assert_close
    assert_close("c128", got, want, al, be, b, a, exact=False)


def test_fxdot_property_against_exact_rationals():
    """Random factors anywhere in the admitted range, drawn by hypothesis
    (where installed): the bound of the exact-sum test holds."""
    hyp = pytest.importorskip("hypothesis")
    st = hyp.strategies

    def in_range(v):
        return v == 0 or 2.0 ** -480 <= abs(v) < 2.0 ** 480

    factor = st.floats(min_value=-(2.0 ** 479), max_value=2.0 ** 479, allow_nan=False,
                       allow_infinity=False).filter(in_range)

    @hyp.settings(max_examples=3000, deadline=None, derandomize=True)
    @hyp.given(st.sampled_from([2, 4]).flatmap(
        lambda n: st.tuples(st.lists(factor, min_size=n, max_size=n), st.lists(factor, min_size=n, max_size=n),
                            st.lists(st.integers(0, 1), min_size=n, max_size=n))))
    def check(case):
        xs, ys, ns = case
        got = costa.costa_debug_fxdot(np.array([xs]), np.array([ys]), np.array([ns], np.int32))[0]
        prods = [Fraction(x) * Fraction(y) * (-1 if k else 1) for x, y, k in zip(xs, ys, ns)]
        exact = sum(prods)
        M = max(abs(p) for p in prods)
        if M == 0:
            assert got == 0.0
            return
        n = len(xs)
        ulp_m = Fraction(math.ulp(float(M)))
        rounded = float(exact)
        bound = n * ulp_m / 128 + (Fraction(math.ulp(rounded)) / 2 if rounded else 0)
        assert abs(Fraction(float(got)) - exact) <= bound

    check()
