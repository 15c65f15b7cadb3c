"""Test helpers for the multi-GPU exchange (costa_exchange_*): processes whose
blocks live in host numpy arenas, and a numpy emulation of the three tile
lists the library plans for each process (pack, local, unpack), applied
through the descriptors' own addresses.

The emulation only moves and combines elements as each descriptor says; with
power-of-two scalars (or beta = 0) its arithmetic is exact, so the result can
be compared with the oracle bit for bit.  It tests the host-side plan: the
partition of tiles between the processes, the package sizes, offsets and
order, and the descriptors' addresses."""
from __future__ import annotations

import ctypes

import numpy as np

from workloads.materialize import HostMatrix, block_element_offsets

TF_TRANSPOSE, TF_FAST, TF_CONJ = 1, 2, 4
_NP = {"f32": np.float32, "f64": np.float64, "c64": np.complex64, "c128": np.complex128}


def block_placement(P: int, G: int) -> np.ndarray:
    """Ranks in contiguous blocks of about P / G per GPU."""
    return np.array([r * G // P for r in range(P)], dtype=np.int32)


def host_ptrs(spec, host: HostMatrix, place, g: int) -> np.ndarray:
    """Block addresses in a host arena; NULL for the blocks of ranks that are
    not on process g."""
    es = host.arena.itemsize
    ptr = (host.arena.ctypes.data + block_element_offsets(spec, host.starts) * es).astype(np.uint64)
    mine = np.asarray(place)[spec.owner] == g
    return np.where(mine, ptr, np.uint64(0))


def aligned_bytes(n: int) -> np.ndarray:
    """A zeroed byte buffer of n bytes starting on a 256-byte boundary."""
    raw = np.zeros(n + 256, dtype=np.uint8)
    off = (-raw.ctypes.data) % 256
    return raw[off:off + n]


def _view(addr: int, dtype, shape, strides):
    es = np.dtype(dtype).itemsize
    span = (shape[0] - 1) * strides[0] + (shape[1] - 1) * strides[1] + es
    buf = (ctypes.c_char * span).from_address(addr)
    return np.ndarray(shape=shape, dtype=dtype, buffer=buf, strides=strides)


def apply_list(tiles, dtype: str, alpha=1.0, beta=0.0, copy: bool = False) -> int:
    """Applies descriptors in the kernel's frame: target (x, y) at
    dst + (x + y * dld), source at src + (x + y * sld), or src + (x * sld + y)
    when transposed; out = alpha * op(b) + beta * a (b conjugated when the
    conjugate flag is set), or a plain copy.  Returns the elements moved."""
    t = _NP[dtype]
    es = np.dtype(t).itemsize
    moved = 0
    for d in tiles:
        nx, ny = int(d["nx"]), int(d["ny"])
        sld, dld, fl = int(d["sld"]), int(d["dld"]), int(d["flags"])
        dst = _view(int(d["dst"]), t, (ny, nx), (dld * es, es))
        if fl & TF_TRANSPOSE:
            src = _view(int(d["src"]), t, (ny, nx), (es, sld * es))
        else:
            src = _view(int(d["src"]), t, (ny, nx), (sld * es, es))
        if copy:
            dst[...] = src
        else:
            b = np.conj(src) if (fl & TF_CONJ) and np.iscomplexobj(src) else src
            if beta == 0:
                dst[...] = (t(alpha) * b).astype(t) if alpha != 1 else b
            else:
                dst[...] = (t(alpha) * b + t(beta) * dst).astype(t)
        moved += nx * ny
    return moved
