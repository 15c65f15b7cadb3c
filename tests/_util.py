"""Test-side helpers that view a layout's buffers as a global matrix.

These rebuild the global m x n matrix block by block with numpy slicing and
reshapes (as_strided over each block's storage).  They are a second,
independent route to the addressing that the oracle does element by element
with binary searches, so the oracle's addressing can be checked against them.
"""
from __future__ import annotations

import numpy as np
from numpy.lib.stride_tricks import as_strided


def block_view(spec, arena_buffers, bi: int, bj: int):
    """Writable numpy view of block (bi, bj) as an h x w matrix."""
    h = int(spec.rsplit[bi + 1] - spec.rsplit[bi])
    w = int(spec.csplit[bj + 1] - spec.csplit[bj])
    buf = arena_buffers[int(spec.buf[bi, bj])]
    off = int(spec.off[bi, bj])
    ld = int(spec.ld[bi, bj])
    es = buf.itemsize
    base = buf[off:]
    if spec.order[bi, bj] == 0:
        strides = (es, ld * es)
    else:
        strides = (ld * es, es)
    return as_strided(base, shape=(h, w), strides=strides)


def global_matrix(spec, arena_buffers) -> np.ndarray:
    out = np.empty((spec.m, spec.n), dtype=arena_buffers[0].dtype if arena_buffers
                   else np.float64)
    for bi in range(spec.nbr):
        r0, r1 = int(spec.rsplit[bi]), int(spec.rsplit[bi + 1])
        for bj in range(spec.nbc):
            c0, c1 = int(spec.csplit[bj]), int(spec.csplit[bj + 1])
            if r1 > r0 and c1 > c0:
                out[r0:r1, c0:c1] = block_view(spec, arena_buffers, bi, bj)
    return out


def scatter_global(spec, arena_buffers, G: np.ndarray) -> None:
    """Write a global matrix into a layout's buffers."""
    for bi in range(spec.nbr):
        r0, r1 = int(spec.rsplit[bi]), int(spec.rsplit[bi + 1])
        for bj in range(spec.nbc):
            c0, c1 = int(spec.csplit[bj]), int(spec.csplit[bj + 1])
            if r1 > r0 and c1 > c0:
                block_view(spec, arena_buffers, bi, bj)[...] = G[r0:r1, c0:c1]


def owner_matrix(spec) -> np.ndarray:
    """Global m x n matrix of owners, by repeating the owners grid."""
    hs = np.diff(spec.rsplit).astype(np.int64)
    ws = np.diff(spec.csplit).astype(np.int64)
    return np.repeat(np.repeat(spec.owner, hs, axis=0), ws, axis=1)


def volume_by_owner_maps(op: str, A_spec, B_spec, P: int) -> np.ndarray:
    """V[p, q] from global owner maps and a bincount."""
    qa = owner_matrix(A_spec)
    ob = owner_matrix(B_spec)
    pb = ob if op == "N" else ob.T
    assert pb.shape == qa.shape
    return np.bincount((pb.astype(np.int64) * P + qa).ravel(),
                       minlength=P * P).reshape(P, P)


def op_apply(op: str, G: np.ndarray) -> np.ndarray:
    if op == "N":
        return G
    if op == "T":
        return G.T
    return np.conj(G.T)


def ulp(x, dtype) -> np.ndarray:
    """Spacing of floating-point numbers at |x| in the real type of dtype."""
    real = np.float32 if dtype in ("f32", "c64") else np.float64
    x = np.abs(np.asarray(x, dtype=real))
    return np.spacing(x)


def tolerance(dtype: str, alpha, beta, bvals, avals, want=None) -> np.ndarray:
    """Per-element, per-component bound on |gpu - oracle| for beta != 0 or
    complex scalars: 2 ulp(M) in the data's precision.

    Real scalars: M = max(|alpha b|, |beta a|).  The kernel computes
    fma(alpha, b, beta * a) and the oracle rounds the exact value once; both
    are roundings of values at most 0.5 ulp(M) apart, so they differ by at
    most 2 ulp(M).

    Complex scalars: M = the largest of the component's product terms
    (2 with beta = 0, 4 otherwise) and of the oracle's value `want`.  The
    oracle uses Dot2 (Ogita, Rump & Oishi 2005) for double data and, for
    float data, a double sum of the exact products rounded once to float:
    within u|x| + gamma_4^2 * sum|terms| of the exact value x.  The kernel
    uses Dot2 in the data's precision (the same bound; the two differ by
    less than 2u|x| + 2 gamma_4^2 * 4M, below 2 ulp(M) plus 2^-45 ulp(M) in
    double and 2^-16 in float); for double data in the middle range
    Kahan's algorithm for two terms (within 2u|x|, Jeannerod, Louvet &
    Muller 2013) or a fixed-point sum on the integer pipes (within 0.5
    ulp(x) + 2^-5 ulp(M), fxdot.h), both under 2 ulp(M) from the oracle.
    The test asserts 2 ulp(M).
    Returned as (re_tol, im_tol) arrays (im_tol zero for real types).
    """
    alpha, beta = complex(alpha), complex(beta)
    b = np.asarray(bvals).astype(np.complex128)
    a = np.asarray(avals).astype(np.complex128)
    if beta == 0:
        a = np.zeros_like(a)
    if alpha.imag == 0 and beta.imag == 0:
        mr = np.maximum(np.abs(alpha.real * b.real), np.abs(beta.real * a.real))
        mi = np.maximum(np.abs(alpha.real * b.imag), np.abs(beta.real * a.imag))
        return 2 * ulp(mr, dtype), 2 * ulp(mi, dtype)
    w = np.zeros_like(b) if want is None else np.asarray(want).astype(np.complex128)
    mr = np.max([np.abs(alpha.real * b.real), np.abs(alpha.imag * b.imag),
                 np.abs(beta.real * a.real), np.abs(beta.imag * a.imag),
                 np.nan_to_num(np.abs(w.real), nan=0.0)], axis=0)
    mi = np.max([np.abs(alpha.real * b.imag), np.abs(alpha.imag * b.real),
                 np.abs(beta.real * a.imag), np.abs(beta.imag * a.real),
                 np.nan_to_num(np.abs(w.imag), nan=0.0)], axis=0)
    return 2 * ulp(mr, dtype), 2 * ulp(mi, dtype)


def _nonfinite_mismatch(g, w):
    """Elements where NaN-ness differs, or where either side is infinite and
    the two are not equal (checked per real component)."""
    bad = np.zeros(g.shape, bool)
    for gc, wc in ((g.real, w.real), (g.imag, w.imag)):
        bad |= np.isnan(gc) != np.isnan(wc)
        inf = np.isinf(gc) | np.isinf(wc)
        bad |= inf & (gc != wc)
    return bad


def max_ulps(dtype, got, want, alpha, beta, bvals, avals) -> float:
    """Largest |gpu - oracle| over the finite elements, in units of the
    bound's 2 ulp(M) / 2 (that is, in ulp(M))."""
    tr, ti = tolerance(dtype, alpha, beta, bvals, avals, want)
    g = np.asarray(got).astype(np.complex128)
    w = np.asarray(want).astype(np.complex128)
    fin = np.isfinite(g) & np.isfinite(w)
    er = np.abs(g.real - w.real)[fin] / (tr[fin] / 2)
    ei = np.abs(g.imag - w.imag)[fin] / np.where(ti[fin] > 0, ti[fin] / 2, 1.0)
    return float(max(np.max(er, initial=0.0), np.max(ei, initial=0.0)))


def assert_close(dtype, got, want, alpha, beta, bvals, avals, exact: bool):
    got = np.asarray(got)
    want = np.asarray(want)
    if exact:
        ok = (got == want) | (np.isnan(got) & np.isnan(want))
        if not np.all(ok):
            k = np.flatnonzero(~ok.ravel())[:5]
            raise AssertionError(f"{(~ok).sum()} mismatches; first at {k}: "
                                 f"got {got.ravel()[k]} want {want.ravel()[k]}")
        return
    g = got.astype(np.complex128)
    w = want.astype(np.complex128)
    nf = _nonfinite_mismatch(g, w)
    if np.any(nf):
        k = np.flatnonzero(nf.ravel())[:5]
        raise AssertionError(f"{nf.sum()} NaN/Inf mismatches; first at {k}: got "
                             f"{got.ravel()[k]} want {want.ravel()[k]}")
    tr, ti = tolerance(dtype, alpha, beta, bvals, avals, want)
    fin = np.isfinite(g) & np.isfinite(w)
    with np.errstate(invalid="ignore"):
        er, ei = np.abs(g.real - w.real), np.abs(g.imag - w.imag)
    bad = fin & ((er > tr) | (ei > ti))
    if np.any(bad):
        k = np.flatnonzero(bad.ravel())[:5]
        raise AssertionError(f"{bad.sum()} out of tolerance; first at {k}: got "
                             f"{got.ravel()[k]} want {want.ravel()[k]} tol {tr.ravel()[k]}")


def exact_case(dtype: str, alpha, beta) -> bool:
    """True when the kernel and the oracle must agree bit for bit: beta == 0
    with a real alpha (one rounding of alpha * b on both sides), or real
    alpha and beta that are both powers of two (both products exact, so the
    kernel's fma and the oracle each round the exact sum once)."""
    alpha, beta = complex(alpha), complex(beta)
    if alpha.imag != 0 or beta.imag != 0:
        return False
    if beta == 0:
        return True
    return all(np.frexp(abs(x.real))[0] == 0.5 for x in (alpha, beta))
