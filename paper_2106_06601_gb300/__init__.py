"""Python binding of the COSTA GB300 library (include/costa_gb300.h).

Argument marshalling only: every step of the reshuffle (overlay, volume,
relabeling, data movement) runs in the native library.  The functions have
the C entry points' names.  Device buffers are passed as integer addresses
(e.g. torch's ``data_ptr()``), streams as ``cudaStream_t`` integers (e.g.
``torch.cuda.current_stream().cuda_stream``).

The library must have been built (``paper_2106_06601_gb300.build.build()``);
importing the binding without it raises ImportError: there is no fallback.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from .build import LIB as _LIB_PATH

COSTA_OK = 0
STATUS_NAMES = {0: "OK", 1: "INVALID_ARG", 2: "LAYOUT", 3: "SHAPE", 4: "DTYPE", 5: "ALLOC",
                6: "CUDA", 7: "INTERNAL"}
DTYPES = {"f32": 0, "f64": 1, "c64": 2, "c128": 3}
OPS = {"N": 0, "T": 1, "C": 2}
MODES = {"direct": 0, "message": 1}
ORDERS = {"C": 0, "R": 1}
_SCALAR_NP = {"f32": np.float32, "f64": np.float64, "c64": np.complex64, "c128": np.complex128}


class CostaError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


class _Block(ctypes.Structure):
    _fields_ = [("ptr", ctypes.c_void_p), ("ld", ctypes.c_int64), ("order", ctypes.c_int32),
                ("reserved", ctypes.c_int32)]


# costa_block as a numpy record, for building block arrays without a Python loop
_BLOCK_DTYPE = np.dtype([("ptr", np.uint64), ("ld", np.int64), ("order", np.int32), ("reserved", np.int32)])
assert _BLOCK_DTYPE.itemsize == ctypes.sizeof(_Block)


class PlanStats(ctypes.Structure):
    _fields_ = [("total_volume", ctypes.c_int64), ("local_identity", ctypes.c_int64),
                ("local_relabeled", ctypes.c_int64), ("n_cells", ctypes.c_int64),
                ("n_tiles", ctypes.c_int64), ("staging_bytes", ctypes.c_int64),
                ("plan_ms", ctypes.c_double), ("volume_ms", ctypes.c_double),
                ("relabel_ms", ctypes.c_double)]

    def as_dict(self):
        return {k: getattr(self, k) for k, _ in self._fields_}


def _load():
    if not os.path.exists(_LIB_PATH):
        raise ImportError(f"COSTA CUDA library not built ({_LIB_PATH}); "
                          "run paper_2106_06601_gb300.build.build()")
    lib = ctypes.CDLL(_LIB_PATH)
    P, I, I64 = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64
    sigs = {
        "costa_layout_create": [P, I, I, I, P, I, P, P, P],
        "costa_layout_create_block_cyclic": [P, I, I64, I64, I64, I64, I, I, ctypes.c_char, P, P, P],
        "costa_layout_destroy": [P],
        "costa_layout_info": [P, P, P, P, P],
        "costa_volume": [P, P, I, P, P],
        "costa_volume_noalloc": [P, P, I, P, P],
        "costa_relabel": [I, P, P, P],
        "costa_transform": [P, P, I, P, P, I, P, P],
        "costa_transform_ex": [P, P, I, P, P, I, P, I, P],
        "costa_transform_batched": [I, P, P, P, P, P, I, P, P],
        "costa_transform_batched_ex": [I, P, P, P, P, P, I, P, I, P],
        "costa_plan_stats_get": [I, P, P, P, I, P, P],
        "costa_release_plans": [],
        "costa_debug_axis_pieces": [P, P, I, I, P, I64, P],
        "costa_volume_grid": [P, P, I, I, P],
        "costa_grid_block_cyclic": [I64, I64, I64, I64, I, I, ctypes.c_char, P, P, P, P, P, P, P, P],
        "costa_relabel_greedy": [I, P, P, P],
        "costa_relabel_cost": [I, P, P, P, P, P, P],
        "costa_layout_create_scalapack": [P, I, P, I64, I64, I64, I64, P],
        "costa_pxgemr2d": [I, I64, I64, P, I64, I64, P, P, I64, I64, P, P],
        "costa_pxtran": [I, I, I64, I64, P, P, I64, I64, P, P, P, I64, I64, P, P],
        "costa_scalapack_release": [],
        "costa_debug_tiles": [P, P, I, P, I64, P],
        "costa_debug_split": [P, P, I, P, I64, P, I64, P, I64, P, P, P],
        "costa_debug_halves": [P, P, I, P, I64, P],
        "costa_debug_groups": [P, P, I, I, P, I64, P],
        "costa_phase_timing": [I],
        "costa_phase_times": [P, P],
        "costa_exchange_sizes": [P, P, I, I, P, I, P, P],
        "costa_exchange_create": [P, P, P, I, I, P, I, P, P],
        "costa_exchange_counts": [P, P, P],
        "costa_exchange_pack": [P, P],
        "costa_exchange_local": [P, P, P, P],
        "costa_exchange_unpack": [P, P, P, P],
        "costa_exchange_destroy": [P],
        "costa_relabel_placement": [I, P, I, P, ctypes.c_double, P, P, P],
        "costa_debug_exchange": [P, P, I, I, P, I, ctypes.c_uint64, ctypes.c_uint64, I, P, I64, P, P],
        "costa_debug_tma": [P, P, I, P],
        "costa_debug_fxdot": [I, I64, P, P, P, P],
    }
    for name, args in sigs.items():
        f = getattr(lib, name)
        f.argtypes = args
        f.restype = ctypes.c_int
    lib.costa_last_error.argtypes = []
    lib.costa_last_error.restype = ctypes.c_char_p
    lib.costa_kernel_launch_count.argtypes = []
    lib.costa_kernel_launch_count.restype = ctypes.c_int64
    lib.costa_abi_version.argtypes = []
    lib.costa_abi_version.restype = ctypes.c_int
    return lib


_lib = _load()


def library():
    """The loaded ctypes library (for symbol checks)."""
    return _lib


def _check(status: int) -> None:
    if status != COSTA_OK:
        raise CostaError(status, _lib.costa_last_error().decode())


def _i64(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.int64)


def _i32(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.int32)


def _p(a: np.ndarray) -> int:
    """Address of an array's data, for a void* argument (the caller keeps the
    array alive across the call)."""
    return a.ctypes.data


class Layout:
    """Owning handle of a costa_layout."""

    def __init__(self, handle: int, dtype: str):
        self.handle = ctypes.c_void_p(handle)
        self.dtype = dtype
        self.nranks = self.info()[2]

    def info(self):
        m, n = ctypes.c_int64(), ctypes.c_int64()
        P, dt = ctypes.c_int(), ctypes.c_int()
        _check(_lib.costa_layout_info(self.handle, ctypes.byref(m), ctypes.byref(n),
                                      ctypes.byref(P), ctypes.byref(dt)))
        return m.value, n.value, P.value, dt.value

    def destroy(self):
        if self.handle:
            _check(_lib.costa_layout_destroy(self.handle))
            self.handle = ctypes.c_void_p(0)

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass


def costa_layout_create(dtype: str, nranks: int, row_splits, col_splits, owners, block_ptrs,
                        block_ld, block_order) -> Layout:
    """Layout from splits, an owners grid and per-block storage (device
    address, leading dimension, order 0 = column-major / 1 = row-major)."""
    R, C = _i64(row_splits), _i64(col_splits)
    nbr, nbc = len(R) - 1, len(C) - 1
    own = _i32(owners).reshape(-1)
    ptrs = np.ascontiguousarray(block_ptrs, dtype=np.uint64).reshape(-1)
    ld = _i64(block_ld).reshape(-1)
    order = _i32(block_order).reshape(-1)
    nblk = nbr * nbc
    assert own.size == nblk and ptrs.size == nblk and ld.size == nblk and order.size == nblk
    blocks = np.zeros(max(1, nblk), dtype=_BLOCK_DTYPE)
    blocks["ptr"][:nblk] = ptrs
    blocks["ld"][:nblk] = ld
    blocks["order"][:nblk] = order
    out = ctypes.c_void_p()
    _check(_lib.costa_layout_create(ctypes.byref(out), DTYPES[dtype], nranks, nbr, _p(R), nbc,
                                    _p(C), _p(own), blocks.ctypes.data))
    return Layout(out.value, dtype)


def costa_layout_create_block_cyclic(dtype: str, m: int, n: int, mb: int, nb: int, pr: int,
                                     pc: int, grid_order: str, rank_perm, rank_ptrs,
                                     lld) -> Layout:
    P = pr * pc
    perm = None if rank_perm is None else _i32(rank_perm)
    ptrs = (ctypes.c_void_p * P)(*[int(x) for x in rank_ptrs])
    lld = _i64(lld)
    out = ctypes.c_void_p()
    _check(_lib.costa_layout_create_block_cyclic(
        ctypes.byref(out), DTYPES[dtype], m, n, mb, nb, pr, pc, grid_order.encode(),
        None if perm is None else _p(perm), ptrs, _p(lld)))
    return Layout(out.value, dtype)


def costa_layout_destroy(layout: Layout) -> None:
    layout.destroy()


def costa_volume(A: Layout, B: Layout, op: str, stream: int = 0) -> np.ndarray:
    """V[p, q]: elements sent from rank p (owner in L(B)) to rank q (owner in L(A))."""
    _, _, P, _ = A.info()
    V = np.zeros((P, P), dtype=np.int64)
    _check(_lib.costa_volume(A.handle, B.handle, OPS[op], _p(V), ctypes.c_void_p(stream)))
    return V


def costa_volume_noalloc(A: Layout, B: Layout, op: str, stream: int = 0) -> np.ndarray:
    """costa_volume without device allocation (fixed 4 MiB scratch)."""
    _, _, P, _ = A.info()
    V = np.zeros((P, P), dtype=np.int64)
    _check(_lib.costa_volume_noalloc(A.handle, B.handle, OPS[op], _p(V), ctypes.c_void_p(stream)))
    return V


def costa_relabel(V):
    """(sigma, local_volume): sigma[q] is the process that takes target label q."""
    V = _i64(V)
    P = V.shape[0]
    sigma = np.zeros(P, dtype=np.int32)
    lv = ctypes.c_int64()
    _check(_lib.costa_relabel(P, _p(V), _p(sigma), ctypes.byref(lv)))
    return sigma, lv.value


def costa_relabel_greedy(V):
    """(sigma, local_volume) from the greedy 2-approximation (Sec. 6)."""
    V = _i64(V)
    P = V.shape[0]
    sigma = np.zeros(P, dtype=np.int32)
    lv = ctypes.c_int64()
    _check(_lib.costa_relabel_greedy(P, _p(V), _p(sigma), ctypes.byref(lv)))
    return sigma, lv.value


def costa_relabel_cost(V, lat, bw):
    """(sigma, W(G), W(G_sigma)) under w = lat + bw * volume for remote packages."""
    V = _i64(V)
    P = V.shape[0]
    lat = np.ascontiguousarray(lat, dtype=np.float64)
    bw = np.ascontiguousarray(bw, dtype=np.float64)
    assert lat.shape == (P, P) and bw.shape == (P, P)
    sigma = np.zeros(P, dtype=np.int32)
    c0, c1 = ctypes.c_double(), ctypes.c_double()
    _check(_lib.costa_relabel_cost(P, _p(V), _p(lat), _p(bw), _p(sigma), ctypes.byref(c0),
                                   ctypes.byref(c1)))
    return sigma, c0.value, c1.value


def costa_relabel_placement(V, G: int, place, intra: float = 0.0):
    """(sigma, W(G), W(G_sigma)) for ranks placed on G GPUs: packages kept
    on their process cost 0, between ranks of one GPU intra * v, between
    GPUs v."""
    V = _i64(V)
    P = V.shape[0]
    pl = _i32(place)
    assert pl.size == P
    sigma = np.zeros(P, dtype=np.int32)
    c0, c1 = ctypes.c_double(), ctypes.c_double()
    _check(_lib.costa_relabel_placement(P, _p(V), G, _p(pl), float(intra), _p(sigma),
                                        ctypes.byref(c0), ctypes.byref(c1)))
    return sigma, c0.value, c1.value


def costa_exchange_sizes(A: Layout, B: Layout, op: str, G: int, place, g: int):
    """(send_bytes[G], recv_bytes[G]) of process g's exchange segments."""
    pl = _i32(place)
    sb, rb = np.zeros(G, np.int64), np.zeros(G, np.int64)
    _check(_lib.costa_exchange_sizes(A.handle, B.handle, OPS[op], G, _p(pl), g, _p(sb), _p(rb)))
    return sb, rb


class Exchange:
    """Owning handle of a costa_exchange: process g's part of the reshuffle
    with the ranks placed on G GPUs.  send_ptr / recv_ptr: device addresses
    of the caller's send and receive buffers."""

    def __init__(self, A: Layout, B: Layout, op: str, G: int, place, g: int, send_ptr: int,
                 recv_ptr: int):
        self.dtype = A.dtype
        self.G = G
        pl = _i32(place)
        out = ctypes.c_void_p()
        _check(_lib.costa_exchange_create(ctypes.byref(out), A.handle, B.handle, OPS[op], G, _p(pl),
                                          g, ctypes.c_void_p(send_ptr), ctypes.c_void_p(recv_ptr)))
        self.handle = out

    def counts(self):
        sb, rb = np.zeros(self.G, np.int64), np.zeros(self.G, np.int64)
        _check(_lib.costa_exchange_counts(self.handle, _p(sb), _p(rb)))
        return sb, rb

    def pack(self, stream: int = 0) -> None:
        _check(_lib.costa_exchange_pack(self.handle, ctypes.c_void_p(stream)))

    def local(self, alpha, beta, stream: int = 0) -> None:
        al, be = _scalar1(self.dtype, alpha), _scalar1(self.dtype, beta)
        _check(_lib.costa_exchange_local(self.handle, ctypes.byref(al), ctypes.byref(be),
                                         ctypes.c_void_p(stream)))

    def unpack(self, alpha, beta, stream: int = 0) -> None:
        al, be = _scalar1(self.dtype, alpha), _scalar1(self.dtype, beta)
        _check(_lib.costa_exchange_unpack(self.handle, ctypes.byref(al), ctypes.byref(be),
                                          ctypes.c_void_p(stream)))

    def destroy(self) -> None:
        if self.handle:
            _check(_lib.costa_exchange_destroy(self.handle))
            self.handle = ctypes.c_void_p(0)

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass


def costa_debug_tma(A: Layout, B: Layout, op: str) -> dict:
    """TMA staging of the plan of (A, B, op) (COSTA_TMA=1 at plan time)."""
    out = np.zeros(6, np.int64)
    _check(_lib.costa_debug_tma(A.handle, B.handle, OPS[op], _p(out)))
    return {"tiles": int(out[0]), "halves_tiles": int(out[1]), "maps": int(out[2]),
            "timeouts": int(out[3]), "kinds": int(out[4]), "halves_kinds": int(out[5])}


def costa_debug_fxdot(x, y, neg) -> np.ndarray:
    """out[k] = sum_i (-1)^neg[k, i] x[k, i] y[k, i] by the kernels' fixed-point
    evaluation of complex-scalar components (host build); x, y, neg: [count, n]
    with n = 2 or 4."""
    x = np.ascontiguousarray(x, dtype=np.float64)
    y = np.ascontiguousarray(y, dtype=np.float64)
    ng = np.ascontiguousarray(neg, dtype=np.int32)
    if x.ndim != 2 or x.shape != y.shape or x.shape != ng.shape:
        raise ValueError("x, y and neg must be [count, n] arrays of one shape")
    out = np.empty(x.shape[0], np.float64)
    _check(_lib.costa_debug_fxdot(x.shape[1], x.shape[0], _p(x), _p(y), _p(ng), _p(out)))
    return out


def costa_debug_exchange(A: Layout, B: Layout, op: str, G: int, place, g: int, send_base: int,
                         recv_base: int, which: str):
    """(descriptors, volumes[2, G]) of process g's pack, local or unpack list."""
    pl = _i32(place)
    w = {"pack": 0, "local": 1, "unpack": 2}[which]
    cnt = ctypes.c_int64()
    vol = np.zeros(2 * G, np.int64)
    _check(_lib.costa_debug_exchange(A.handle, B.handle, OPS[op], G, _p(pl), g, send_base,
                                     recv_base, w, None, 0, ctypes.byref(cnt), _p(vol)))
    out = np.zeros(max(1, cnt.value), dtype=TILE_DTYPE)
    _check(_lib.costa_debug_exchange(A.handle, B.handle, OPS[op], G, _p(pl), g, send_base,
                                     recv_base, w, _p(out), cnt.value, ctypes.byref(cnt), None))
    return out[:cnt.value], vol.reshape(2, G)


class _BlacsGrid(ctypes.Structure):
    _fields_ = [("nprow", ctypes.c_int), ("npcol", ctypes.c_int), ("order", ctypes.c_char),
                ("local", ctypes.c_void_p), ("lld", ctypes.c_void_p)]


class BlacsGrid:
    """A grid of virtual ranks with one column-major local matrix each
    (costa_blacs_grid): device addresses and leading dimensions per rank."""

    def __init__(self, nprow: int, npcol: int, order: str, local_ptrs, lld=None):
        P = nprow * npcol
        self.ptrs = (ctypes.c_void_p * P)(*[int(x) for x in local_ptrs])
        self.lld = None if lld is None else _i64(lld)
        self.s = _BlacsGrid(nprow, npcol, order.encode(), ctypes.cast(self.ptrs, ctypes.c_void_p),
                            None if self.lld is None else self.lld.ctypes.data)

    def ref(self):
        return ctypes.byref(self.s)


def costa_layout_create_scalapack(dtype: str, grid: BlacsGrid, i: int, j: int, m: int, n: int,
                                  desc) -> Layout:
    d = _i64(desc)
    out = ctypes.c_void_p()
    _check(_lib.costa_layout_create_scalapack(ctypes.byref(out), DTYPES[dtype], grid.ref(), i, j,
                                              m, n, _p(d)))
    return Layout(out.value, dtype)


def costa_pxgemr2d(dtype: str, m: int, n: int, ga: BlacsGrid, ia: int, ja: int, desca,
                   gb: BlacsGrid, ib: int, jb: int, descb, stream: int = 0) -> None:
    """sub(B) := sub(A) (ScaLAPACK PxGEMR2D; 1-based ia, ja, ib, jb)."""
    da, db = _i64(desca), _i64(descb)
    _check(_lib.costa_pxgemr2d(DTYPES[dtype], m, n, ga.ref(), ia, ja, _p(da), gb.ref(), ib, jb,
                               _p(db), ctypes.c_void_p(stream)))


def costa_pxtran(dtype: str, m: int, n: int, alpha, ga: BlacsGrid, ia: int, ja: int, desca, beta,
                 gc: BlacsGrid, ic: int, jc: int, descc, conjugate: bool = False,
                 stream: int = 0) -> None:
    """sub(C) := beta sub(C) + alpha op(sub(A)), op = T (PxTRAN) or C (PxTRANC)."""
    da, dc = _i64(desca), _i64(descc)
    al, be = _scalars(dtype, [alpha]), _scalars(dtype, [beta])
    _check(_lib.costa_pxtran(DTYPES[dtype], int(conjugate), m, n, _p(al), ga.ref(), ia, ja,
                             _p(da), _p(be), gc.ref(), ic, jc, _p(dc), ctypes.c_void_p(stream)))


def costa_scalapack_release() -> None:
    _check(_lib.costa_scalapack_release())


class _GridDesc(ctypes.Structure):
    _fields_ = [("nbr", ctypes.c_int), ("nbc", ctypes.c_int), ("row_splits", ctypes.c_void_p),
                ("row_procs", ctypes.c_void_p), ("col_splits", ctypes.c_void_p),
                ("col_procs", ctypes.c_void_p), ("pr", ctypes.c_int), ("pc", ctypes.c_int),
                ("grid", ctypes.c_void_p)]


class GridLayout:
    """A process-grid layout without per-block arrays (costa_grid_desc)."""

    def __init__(self, row_splits, row_procs, col_splits, col_procs, grid):
        self.rs, self.cs = _i64(row_splits), _i64(col_splits)
        self.rp, self.cp = _i32(row_procs), _i32(col_procs)
        self.grid = _i32(grid)
        assert self.grid.ndim == 2
        self.desc = _GridDesc(len(self.rs) - 1, len(self.cs) - 1, self.rs.ctypes.data,
                              self.rp.ctypes.data, self.cs.ctypes.data, self.cp.ctypes.data,
                              self.grid.shape[0], self.grid.shape[1], self.grid.ctypes.data)

    @staticmethod
    def block_cyclic(m, n, mb, nb, pr, pc, grid_order="R", rank_perm=None):
        """The grid of a block-cyclic layout (costa_grid_block_cyclic)."""
        nbr, nbc = ctypes.c_int(), ctypes.c_int()
        perm = None if rank_perm is None else _i32(rank_perm)
        args = (m, n, mb, nb, pr, pc, grid_order.encode(), None if perm is None else _p(perm))
        _check(_lib.costa_grid_block_cyclic(*args, None, None, None, None, None,
                                            ctypes.byref(nbr), ctypes.byref(nbc)))
        rs, cs = np.zeros(nbr.value + 1, np.int64), np.zeros(nbc.value + 1, np.int64)
        rp, cp = np.zeros(max(1, nbr.value), np.int32), np.zeros(max(1, nbc.value), np.int32)
        grid = np.zeros((pr, pc), np.int32)
        _check(_lib.costa_grid_block_cyclic(*args, _p(rs), _p(rp), _p(cs), _p(cp), _p(grid),
                                            ctypes.byref(nbr), ctypes.byref(nbc)))
        return GridLayout(rs, rp[:nbr.value], cs, cp[:nbc.value], grid)


def costa_volume_grid(A: GridLayout, B: GridLayout, op: str, P: int) -> np.ndarray:
    """V[p, q] for process-grid layouts from 1-D overlaps (no device work)."""
    V = np.zeros((P, P), dtype=np.int64)
    _check(_lib.costa_volume_grid(ctypes.byref(A.desc), ctypes.byref(B.desc), OPS[op], P, _p(V)))
    return V


def _scalars(dtype: str, values) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(values, dtype=_SCALAR_NP[dtype]).reshape(-1))


# One host scalar of each element type as a ctypes value (real, or re/im pair).
_SCALAR_CT = {"f32": ctypes.c_float, "f64": ctypes.c_double,
              "c64": ctypes.c_float * 2, "c128": ctypes.c_double * 2}


def _scalar1(dtype: str, v):
    if dtype in ("f32", "f64"):
        return _SCALAR_CT[dtype](v)
    v = complex(v)
    return _SCALAR_CT[dtype](v.real, v.imag)


def costa_transform(A: Layout, B: Layout, op: str, alpha, beta, relabel: bool = False,
                    stream: int = 0, mode: str = "direct") -> np.ndarray:
    """A = alpha * op(B) + beta * A, asynchronous on `stream`; returns sigma."""
    sigma = np.zeros(A.nranks, dtype=np.int32)
    al, be = _scalar1(A.dtype, alpha), _scalar1(A.dtype, beta)
    _check(_lib.costa_transform_ex(A.handle, B.handle, OPS[op], ctypes.byref(al), ctypes.byref(be),
                                   int(relabel), sigma.ctypes.data, MODES[mode], stream))
    return sigma


def costa_transform_batched(As, Bs, ops, alphas, betas, relabel: bool = False,
                            stream: int = 0, mode: str = "direct") -> np.ndarray:
    n = len(As)
    _, _, P, _ = As[0].info()
    sigma = np.zeros(P, dtype=np.int32)
    ha = (ctypes.c_void_p * n)(*[a.handle.value for a in As])
    hb = (ctypes.c_void_p * n)(*[b.handle.value for b in Bs])
    op = _i32([OPS[o] for o in ops])
    al, be = _scalars(As[0].dtype, alphas), _scalars(As[0].dtype, betas)
    assert al.size == n and be.size == n
    _check(_lib.costa_transform_batched_ex(n, ha, hb, _p(op), _p(al), _p(be), int(relabel),
                                           _p(sigma), MODES[mode], ctypes.c_void_p(stream)))
    return sigma


def costa_plan_stats_get(As, Bs, ops, relabel: bool = False, stream: int = 0) -> dict:
    if isinstance(As, Layout):
        As, Bs, ops = [As], [Bs], [ops]
    n = len(As)
    ha = (ctypes.c_void_p * n)(*[a.handle.value for a in As])
    hb = (ctypes.c_void_p * n)(*[b.handle.value for b in Bs])
    op = _i32([OPS[o] for o in ops])
    st = PlanStats()
    _check(_lib.costa_plan_stats_get(n, ha, hb, _p(op), int(relabel), ctypes.byref(st),
                                     ctypes.c_void_p(stream)))
    return st.as_dict()


def costa_release_plans() -> None:
    _check(_lib.costa_release_plans())


def costa_last_error() -> str:
    return _lib.costa_last_error().decode()


def costa_kernel_launch_count() -> int:
    return _lib.costa_kernel_launch_count()


def costa_abi_version() -> int:
    return _lib.costa_abi_version()


def costa_phase_timing(enable: bool) -> None:
    """Turns per-phase CUDA-event timing of transform calls on or off."""
    _check(_lib.costa_phase_timing(int(bool(enable))))


def costa_phase_times() -> list:
    """Device milliseconds of the phases of the last timed transform call on
    the current device: [remap] (direct mode) or [pack, local, unpack]
    (message mode).  Waits for that call's events."""
    ms = (ctypes.c_double * 3)()
    n = ctypes.c_int(0)
    _check(_lib.costa_phase_times(ms, ctypes.byref(n)))
    return [ms[k] for k in range(n.value)]


def costa_layout_from_spec(spec, dtype: str, block_ptrs) -> Layout:
    """costa_layout_create from any object with the fields rsplit, csplit,
    owner, nranks, ld, order (one entry per block) and per-block device
    addresses `block_ptrs`."""
    return costa_layout_create(dtype, spec.nranks, spec.rsplit, spec.csplit, spec.owner,
                               block_ptrs, spec.ld, spec.order)


def costa_debug_axis_pieces(A: Layout, B: Layout, op: str, axis: int) -> np.ndarray:
    """The plan's pieces of one axis of A, as an int32 array [count, 6]."""
    cnt = ctypes.c_int64()
    _check(_lib.costa_debug_axis_pieces(A.handle, B.handle, OPS[op], axis, None, 0,
                                        ctypes.byref(cnt)))
    out = np.zeros((max(1, cnt.value), 6), dtype=np.int32)
    _check(_lib.costa_debug_axis_pieces(A.handle, B.handle, OPS[op], axis, _p(out), cnt.value,
                                        ctypes.byref(cnt)))
    return out[:cnt.value]


TILE_DTYPE = np.dtype([("src", np.uint64), ("dst", np.uint64), ("sld", np.int32),
                       ("dld", np.int32), ("nx", np.uint16), ("ny", np.uint16),
                       ("prob", np.uint16), ("flags", np.uint16)])


def costa_debug_split(A: Layout, B: Layout, op: str):
    """(full-size tiles, one-pass pieces, group offsets) of the direct list."""
    nt, npc, ng = ctypes.c_int64(), ctypes.c_int64(), ctypes.c_int64()
    _check(_lib.costa_debug_split(A.handle, B.handle, OPS[op], None, 0, None, 0, None, 0,
                                  ctypes.byref(nt), ctypes.byref(npc), ctypes.byref(ng)))
    tiles = np.zeros(max(1, nt.value), dtype=TILE_DTYPE)
    pieces = np.zeros(max(1, npc.value), dtype=TILE_DTYPE)
    ngo = ng.value + 1 if ng.value > 0 else 0
    groups = np.zeros(max(1, ngo), dtype=np.uint32)
    _check(_lib.costa_debug_split(A.handle, B.handle, OPS[op], tiles.ctypes.data, nt.value,
                                  pieces.ctypes.data, npc.value, groups.ctypes.data, ngo,
                                  ctypes.byref(nt), ctypes.byref(npc), ctypes.byref(ng)))
    return tiles[:nt.value], pieces[:npc.value], groups[:ngo]


def costa_debug_groups(A: Layout, B: Layout, op: str, reads_a: bool) -> np.ndarray:
    """Group offsets of the small-tile pieces for one class of kinds."""
    cnt = ctypes.c_int64()
    _check(_lib.costa_debug_groups(A.handle, B.handle, OPS[op], int(reads_a), None, 0, ctypes.byref(cnt)))
    n = cnt.value + 1 if cnt.value > 0 else 0
    out = np.zeros(max(1, n), dtype=np.uint32)
    _check(_lib.costa_debug_groups(A.handle, B.handle, OPS[op], int(reads_a), out.ctypes.data, n,
                                   ctypes.byref(cnt)))
    return out[:n]


def costa_debug_halves(A: Layout, B: Layout, op: str) -> np.ndarray:
    """The aligned tiles as x-halves (empty when the pair has no halves list)."""
    cnt = ctypes.c_int64()
    _check(_lib.costa_debug_halves(A.handle, B.handle, OPS[op], None, 0, ctypes.byref(cnt)))
    out = np.zeros(max(1, cnt.value), dtype=TILE_DTYPE)
    _check(_lib.costa_debug_halves(A.handle, B.handle, OPS[op], out.ctypes.data, cnt.value,
                                   ctypes.byref(cnt)))
    return out[:cnt.value]


def costa_debug_tiles(A: Layout, B: Layout, op: str) -> np.ndarray:
    """The direct-mode tile list of (A, B, op) as a structured array."""
    cnt = ctypes.c_int64()
    _check(_lib.costa_debug_tiles(A.handle, B.handle, OPS[op], None, 0, ctypes.byref(cnt)))
    out = np.zeros(max(1, cnt.value), dtype=TILE_DTYPE)
    _check(_lib.costa_debug_tiles(A.handle, B.handle, OPS[op], out.ctypes.data, cnt.value,
                                  ctypes.byref(cnt)))
    return out[:cnt.value]
