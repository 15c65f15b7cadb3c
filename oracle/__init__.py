"""CPU oracle (test infrastructure only).

Only the tests, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline and
reference legs may import this package.  It shares no code with the CUDA
library.  The C source (costa_oracle.c) holds the per-element definitions and
their citations; this module builds it with gcc and marshals numpy arrays.

Functions that have no independent pin are marked "parity unpinned" in their
docstring; every function here is pinned by tests/test_oracle_pins.py.
"""
from __future__ import annotations

import contextlib
import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "costa_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB = os.path.join(_BUILD, "liboracle.so")

DTYPES = {"f32": 0, "f64": 1, "c64": 2, "c128": 3}
OPS = {"N": 0, "T": 1, "C": 2}
_NP = {"f32": np.float32, "f64": np.float64, "c64": np.complex64, "c128": np.complex128}

_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle into oracle/_build/liboracle.so (gcc, OpenMP)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-ffp-contract=off", "-fno-fast-math",
               "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB)
    return _LIB


class _OLayout(ctypes.Structure):
    _fields_ = [("nbr", ctypes.c_int64), ("nbc", ctypes.c_int64),
                ("rsplit", ctypes.c_void_p), ("csplit", ctypes.c_void_p),
                ("owner", ctypes.c_void_p), ("buf", ctypes.c_void_p),
                ("off", ctypes.c_void_p), ("ld", ctypes.c_void_p),
                ("order", ctypes.c_void_p)]


def _bind(cdll):
    P = ctypes.c_void_p
    cdll.oracle_transform.argtypes = [ctypes.c_int, ctypes.c_int, P, P, P, P, P, P,
                                      ctypes.c_int64, ctypes.c_int64, ctypes.c_int]
    cdll.oracle_transform.restype = ctypes.c_int
    cdll.oracle_volume.argtypes = [ctypes.c_int, P, P, ctypes.c_int, P, ctypes.c_int]
    cdll.oracle_volume.restype = ctypes.c_int
    cdll.oracle_locate_many.argtypes = [P, ctypes.c_int64, P, P, P, P]
    cdll.oracle_combine_many.argtypes = [ctypes.c_int, ctypes.c_int, P, P,
                                         ctypes.c_int64, P, P, P]
    cdll.oracle_lap_bruteforce.argtypes = [ctypes.c_int, P, P]
    cdll.oracle_lap_bruteforce.restype = ctypes.c_int64
    cdll.oracle_lap_subset_dp.argtypes = [ctypes.c_int, P, P]
    cdll.oracle_lap_subset_dp.restype = ctypes.c_int64
    cdll.oracle_lap_greedy.argtypes = [ctypes.c_int, P, P]
    cdll.oracle_lap_greedy.restype = ctypes.c_int64
    cdll.oracle_cost_W.argtypes = [ctypes.c_int, P, P, P, P]
    cdll.oracle_cost_W.restype = ctypes.c_double
    cdll.oracle_copr_bruteforce_cost.argtypes = [ctypes.c_int, P, P, P, P]
    cdll.oracle_copr_bruteforce_cost.restype = ctypes.c_double
    return cdll


def lib():
    global _lib
    with _lock:
        if _lib is None:
            _lib = _bind(ctypes.CDLL(build()))
        return _lib


def compile_variant(source_text: str, out_path: str) -> str:
    """Compiles a modified copy of costa_oracle.c with the oracle's own flags.
    Test hook: the planted-mistake tests build mutated oracles with it."""
    src = out_path + ".c"
    with open(src, "w") as f:
        f.write(source_text)
    cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-ffp-contract=off", "-fno-fast-math",
           "-fPIC", "-shared", "-o", out_path, src, "-lm"]
    subprocess.run(cmd, check=True)
    return out_path


def source_text() -> str:
    with open(_SRC) as f:
        return f.read()


@contextlib.contextmanager
def loaded(path: str):
    """Runs this module's functions on another build of the oracle (a mutated
    copy from compile_variant) inside the block.  Test hook only."""
    global _lib
    lib()
    with _lock:
        saved = _lib
        _lib = _bind(ctypes.CDLL(path))
    try:
        yield
    finally:
        with _lock:
            _lib = saved


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


class _Layout:
    """Keeps the int arrays of a layout alive while C reads them."""

    def __init__(self, spec):
        self.arrays = [np.ascontiguousarray(spec.rsplit, np.int64),
                       np.ascontiguousarray(spec.csplit, np.int64),
                       np.ascontiguousarray(spec.owner, np.int32),
                       np.ascontiguousarray(spec.buf, np.int32),
                       np.ascontiguousarray(spec.off, np.int64),
                       np.ascontiguousarray(spec.ld, np.int64),
                       np.ascontiguousarray(spec.order, np.int32)]
        a = self.arrays
        self.s = _OLayout(spec.nbr, spec.nbc, *[x.ctypes.data for x in a])

    def ref(self):
        return ctypes.byref(self.s)


def scalar(dtype: str, x) -> complex:
    """A scalar in the matrix's own type (alpha and beta are of A's dtype):
    rounded to float32 for f32/c64 data."""
    z = complex(x)
    if dtype in ("f32", "c64"):
        return complex(float(np.float32(z.real)), float(np.float32(z.imag)))
    return z


def _scalar(dtype: str, x) -> np.ndarray:
    z = scalar(dtype, x)
    return np.array([z.real, z.imag], dtype=np.float64)


def default_threads() -> int:
    return os.cpu_count() or 1


def transform(dtype: str, op: str, alpha, beta, A_spec, A_bufs, B_spec, B_bufs,
              rows=None, threads: int | None = None) -> None:
    """In place on the numpy buffers A_bufs: A <- alpha op(B) + beta A (Eq. 1),
    element by element, for target rows `rows` = (begin, end) of A (all rows
    by default)."""
    for b in list(A_bufs) + list(B_bufs):
        assert b.dtype == _NP[dtype] and b.flags.c_contiguous
    la, lb = _Layout(A_spec), _Layout(B_spec)
    abufs = (ctypes.c_void_p * max(1, len(A_bufs)))(*[b.ctypes.data for b in A_bufs])
    bbufs = (ctypes.c_void_p * max(1, len(B_bufs)))(*[b.ctypes.data for b in B_bufs])
    r0, r1 = (0, A_spec.m) if rows is None else rows
    al, be = _scalar(dtype, alpha), _scalar(dtype, beta)
    rc = lib().oracle_transform(DTYPES[dtype], OPS[op], _ptr(al), _ptr(be), la.ref(),
                                abufs, lb.ref(), bbufs, r0, r1,
                                threads or default_threads())
    if rc != 0:
        raise ValueError("oracle_transform: shape mismatch")


def volume(op: str, A_spec, B_spec, P: int, threads: int | None = None) -> np.ndarray:
    """V[p, q]: elements whose source is owned by p in L(B) and whose target
    is owned by q in L(A), counted element by element (Alg. 2's S_pq sizes)."""
    V = np.zeros((P, P), dtype=np.int64)
    la, lb = _Layout(A_spec), _Layout(B_spec)
    rc = lib().oracle_volume(OPS[op], la.ref(), lb.ref(), P, _ptr(V),
                             threads or default_threads())
    if rc != 0:
        raise ValueError("oracle_volume: shape mismatch")
    return V


def locate(spec, ij: np.ndarray):
    """(owner, buffer, element offset) of each (i, j) row of ij in a layout."""
    ij = np.ascontiguousarray(ij, dtype=np.int64).reshape(-1, 2)
    n = ij.shape[0]
    owner = np.empty(n, np.int32)
    buf = np.empty(n, np.int32)
    off = np.empty(n, np.int64)
    l = _Layout(spec)
    lib().oracle_locate_many(l.ref(), n, _ptr(ij), _ptr(owner), _ptr(buf), _ptr(off))
    return owner, buf, off


def combine(dtype: str, op: str, alpha, beta, bvals: np.ndarray, avals: np.ndarray):
    """alpha * op(b) + beta * a element-wise, for values already gathered."""
    bvals = np.ascontiguousarray(bvals, dtype=_NP[dtype])
    avals = np.ascontiguousarray(avals, dtype=_NP[dtype])
    out = np.empty_like(bvals)
    al, be = _scalar(dtype, alpha), _scalar(dtype, beta)
    lib().oracle_combine_many(DTYPES[dtype], OPS[op], _ptr(al), _ptr(be), bvals.size,
                              _ptr(bvals), _ptr(avals), _ptr(out))
    return out


def objective(V: np.ndarray, sigma) -> int:
    """sum_q V[sigma(q), q]: the volume that stays local under sigma."""
    V = np.asarray(V)
    return int(sum(int(V[int(sigma[q]), q]) for q in range(V.shape[0])))


def lap_bruteforce(V: np.ndarray):
    """Optimal relabeling by enumerating all P! permutations (P <= 12)."""
    V = np.ascontiguousarray(V, dtype=np.int64)
    P = V.shape[0]
    sigma = np.zeros(P, dtype=np.int32)
    best = lib().oracle_lap_bruteforce(P, _ptr(V), _ptr(sigma))
    return int(best), sigma


def lap_subset_dp(V: np.ndarray):
    """Optimal relabeling by dynamic programming over subsets (P <= 24)."""
    V = np.ascontiguousarray(V, dtype=np.int64)
    P = V.shape[0]
    sigma = np.zeros(P, dtype=np.int32)
    best = lib().oracle_lap_subset_dp(P, _ptr(V), _ptr(sigma))
    return int(best), sigma


def lap_greedy(V: np.ndarray):
    """The greedy relabeling of Sec. 6 (a 2-approximation): pairs by
    decreasing volume (ties: smaller p, then smaller q), each kept when both
    ends are free; leftover labels take leftover processes in order."""
    V = np.ascontiguousarray(V, dtype=np.int64)
    P = V.shape[0]
    sigma = np.zeros(P, dtype=np.int32)
    total = lib().oracle_lap_greedy(P, _ptr(V), _ptr(sigma))
    return int(total), sigma


def cost_W(V, lat, bw, sigma) -> float:
    """W(G_sigma) under w = lat + bw * volume for remote non-empty packages
    (Def. RG, Eq. WG)."""
    V = np.ascontiguousarray(V, dtype=np.int64)
    lat = np.ascontiguousarray(lat, dtype=np.float64)
    bw = np.ascontiguousarray(bw, dtype=np.float64)
    sig = np.ascontiguousarray(sigma, dtype=np.int32)
    return float(lib().oracle_cost_W(V.shape[0], _ptr(V), _ptr(lat), _ptr(bw), _ptr(sig)))


def copr_bruteforce_cost(V, lat, bw):
    """(min W(G_sigma), sigma) over all permutations (P <= 10), Def. COPR."""
    V = np.ascontiguousarray(V, dtype=np.int64)
    lat = np.ascontiguousarray(lat, dtype=np.float64)
    bw = np.ascontiguousarray(bw, dtype=np.float64)
    P = V.shape[0]
    sigma = np.zeros(P, dtype=np.int32)
    best = lib().oracle_copr_bruteforce_cost(P, _ptr(V), _ptr(lat), _ptr(bw), _ptr(sigma))
    return float(best), sigma


def lap_library(V: np.ndarray):
    """Optimal relabeling by scipy's linear_sum_assignment (maximize); exact
    for integer weights below 2**53."""
    from scipy.optimize import linear_sum_assignment
    V = np.asarray(V, dtype=np.int64)
    assert int(V.sum()) < 2 ** 53
    p, q = linear_sum_assignment(V.astype(np.float64), maximize=True)
    sigma = np.empty(V.shape[0], dtype=np.int32)
    sigma[q] = p
    return objective(V, sigma), sigma


def lap_optimum(V: np.ndarray) -> int:
    """The optimal local volume max_sigma sum_q V[sigma(q), q]."""
    P = np.asarray(V).shape[0]
    if P <= 8:
        return lap_bruteforce(V)[0]
    if P <= 20:
        return lap_subset_dp(V)[0]
    return lap_library(V)[0]
