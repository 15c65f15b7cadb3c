"""Host and device buffers for a Problem (allocation and filling only).

Every buffer of a layout (normally one per virtual rank) becomes a slice of one
arena: a flat host (numpy) or device (torch) array in which each buffer starts
on a 256-byte boundary, optionally with guard elements before and after it.
The arena's guard and padding elements can be pre-set to a sentinel so that a
test can check that nothing outside the blocks was written.
"""
from __future__ import annotations

import numpy as np

from . import gen

ALIGN_BYTES = 256

_TORCH_TYPES = {"f32": "float32", "f64": "float64", "c64": "complex64",
                "c128": "complex128"}
ESIZE = {"f32": 4, "f64": 8, "c64": 8, "c128": 16}


def torch_dtype(dtype: str):
    import torch
    return getattr(torch, _TORCH_TYPES[dtype])


def arena_offsets(bufsize, esize: int, guard: int = 0):
    """Element offset of each buffer inside an arena, and the arena length."""
    align = max(1, ALIGN_BYTES // esize)
    starts = []
    pos = 0
    for sz in bufsize:
        pos += guard
        pos = (pos + align - 1) // align * align
        starts.append(pos)
        pos += int(sz) + guard
    total = (pos + align - 1) // align * align
    return np.array(starts, dtype=np.int64), max(total, align)


def block_element_offsets(spec, starts) -> np.ndarray:
    """Arena element offset of each block's (0, 0) entry, [nbr, nbc] int64."""
    return starts[spec.buf] + spec.off


def value_kind_fill_np(out, dtype, kind, seed, stream):
    if kind == "nan":
        out[...] = np.nan if dtype in ("f32", "f64") else complex(np.nan, np.nan)
        return out
    return gen.fill_np(out, dtype, kind, seed, stream)


class HostMatrix:
    """A layout's buffers in one numpy arena."""

    def __init__(self, spec, dtype: str, guard: int = 0, sentinel=None):
        self.spec, self.dtype, self.guard = spec, dtype, guard
        self.starts, total = arena_offsets(spec.bufsize, ESIZE[dtype], guard)
        # zeroed (or sentinel-filled) so that alignment gaps are deterministic
        self.arena = np.zeros(total, dtype=gen.np_dtype(dtype))
        if sentinel is not None:
            self.arena[...] = sentinel

    def buffer(self, r: int) -> np.ndarray:
        s = int(self.starts[r])
        return self.arena[s:s + int(self.spec.bufsize[r])]

    def buffers(self) -> list:
        return [self.buffer(r) for r in range(self.spec.nbuf)]

    def fill(self, kind: str, seed: int, stream_of) -> "HostMatrix":
        for r in range(self.spec.nbuf):
            value_kind_fill_np(self.buffer(r), self.dtype, kind, seed, stream_of(r))
        return self

    def copy(self) -> "HostMatrix":
        h = HostMatrix.__new__(HostMatrix)
        h.spec, h.dtype, h.guard, h.starts = self.spec, self.dtype, self.guard, self.starts
        h.arena = self.arena.copy()
        return h


class DeviceMatrix:
    """A layout's buffers in one torch arena on a device."""

    def __init__(self, spec, dtype: str, device, guard: int = 0, sentinel=None):
        import torch
        self.spec, self.dtype, self.guard = spec, dtype, guard
        self.esize = ESIZE[dtype]
        self.starts, total = arena_offsets(spec.bufsize, self.esize, guard)
        self.arena = torch.empty(total, dtype=torch_dtype(dtype), device=device)
        if sentinel is not None:
            self.arena.fill_(sentinel)

    def buffer(self, r: int):
        s = int(self.starts[r])
        return self.arena[s:s + int(self.spec.bufsize[r])]

    def block_ptrs(self) -> np.ndarray:
        base = self.arena.data_ptr()
        off = block_element_offsets(self.spec, self.starts)
        return (base + off * self.esize).astype(np.uint64)

    def upload(self, host: HostMatrix) -> "DeviceMatrix":
        import torch
        assert host.arena.size == self.arena.numel()
        self.arena.copy_(torch.from_numpy(host.arena))
        return self

    def download(self) -> HostMatrix:
        h = HostMatrix.__new__(HostMatrix)
        h.spec, h.dtype, h.guard, h.starts = self.spec, self.dtype, self.guard, self.starts
        h.arena = self.arena.cpu().numpy()
        return h

    def fill(self, kind: str, seed: int, stream_of) -> "DeviceMatrix":
        for r in range(self.spec.nbuf):
            b = self.buffer(r)
            if kind == "nan":
                b.fill_(float("nan") if self.dtype in ("f32", "f64")
                        else complex(float("nan"), float("nan")))
            else:
                gen.fill_torch(b, self.dtype, kind, seed, stream_of(r))
        return self


def host_problem(prob, guard: int = 0, sentinel=None):
    """(B, A) host matrices of a problem, filled from its value streams."""
    B = HostMatrix(prob.B, prob.dtype, guard, sentinel).fill(prob.b_kind, prob.seed,
                                                            prob.src_stream)
    A = HostMatrix(prob.A, prob.dtype, guard, sentinel).fill(prob.a_kind, prob.seed,
                                                            prob.tgt_stream)
    return B, A
