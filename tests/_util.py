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


def tolerance(dtype: str, alpha, beta, bvals, avals) -> np.ndarray:
    """Per-element, per-component bound on |gpu - oracle| for beta != 0 or
    complex scalars.

    Real scalars: the kernel computes fma(alpha, b, beta * a); the oracle
    rounds the exact value once.  Both results are roundings of values at most
    0.5 ulp(M) apart, M = max(|alpha b|, |beta a|), so they differ by at most
    2 ulp(M).  Complex scalars with non-zero imaginary parts: each component
    is a chain of up to four fma/mul roundings, each off by at most
    0.5 ulp(S), S = sum of |terms|, and the oracle by 0.5 ulp(S): 3 ulp(S).
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
    sr = (np.abs(alpha.real * b.real) + np.abs(alpha.imag * b.imag)
          + np.abs(beta.real * a.real) + np.abs(beta.imag * a.imag))
    si = (np.abs(alpha.real * b.imag) + np.abs(alpha.imag * b.real)
          + np.abs(beta.real * a.imag) + np.abs(beta.imag * a.real))
    return 3 * ulp(sr, dtype), 3 * ulp(si, dtype)


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
    tr, ti = tolerance(dtype, alpha, beta, bvals, avals)
    g = got.astype(np.complex128)
    w = want.astype(np.complex128)
    er, ei = np.abs(g.real - w.real), np.abs(g.imag - w.imag)
    bad = (er > tr) | (ei > ti)
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
