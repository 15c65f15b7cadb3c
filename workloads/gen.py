"""Seeded, counter-based value generator for synthetic matrices.

This module produces input numbers only; it contains none of the reshuffle
arithmetic.  Both the CUDA path and the CPU oracle receive buffers filled from
here.

Definition (SplitMix64, Steele, Lea & Flood, "Fast splittable pseudorandom
number generators", OOPSLA 2014): a stream with 64-bit state s0 yields, as its
k-th draw (k = 0, 1, ...),

    z = s0 + (k + 1) * GAMMA              (mod 2**64)
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9
    z = (z ^ (z >> 27)) * 0x94D049BB133111EB
    draw = z ^ (z >> 31)

so any draw can be computed from its index alone.  The state of stream
``stream`` under ``seed`` is ``mix(seed + stream * STREAM_MUL)``.

Value maps:
  uniform[-1, 1), f64:  (draw >> 11) * 2**-52 - 1     (exact in f64)
  uniform[-1, 1), f32:  (draw >> 40) * 2**-23 - 1     (exact in f32)
  normal(0, 1):         Box-Muller, r * cos(2 pi u2) with
                        u1 = ((d0 >> 11) + 1) * 2**-53, u2 = (d1 >> 11) * 2**-53
Element k of a real buffer uses draw k (uniform) or draws 2k, 2k+1 (normal).
Element k of a complex buffer takes its real part from the real-valued
sequence at index 2k and its imaginary part from index 2k+1.

A numpy implementation (host) and a torch implementation (any device) are
given; they agree bit for bit on the integer draws and on the uniform maps.
"""
from __future__ import annotations

import numpy as np

GAMMA = 0x9E3779B97F4A7C15
MUL1 = 0xBF58476D1CE4E5B9
MUL2 = 0x94D049BB133111EB
STREAM_MUL = 0xD1B54A32D192ED03
MASK64 = (1 << 64) - 1

_CHUNK = 1 << 24


def _mix_int(z: int) -> int:
    z &= MASK64
    z = ((z ^ (z >> 30)) * MUL1) & MASK64
    z = ((z ^ (z >> 27)) * MUL2) & MASK64
    return z ^ (z >> 31)


def stream_state(seed: int, stream: int) -> int:
    """64-bit starting state of one stream."""
    return _mix_int((seed + stream * STREAM_MUL) & MASK64)


def draw_int(seed: int, stream: int, k: int) -> int:
    """The k-th 64-bit draw of a stream, as a Python int (reference form)."""
    return _mix_int(stream_state(seed, stream) + (k + 1) * GAMMA)


# ----------------------------------------------------------------------------
# numpy (host)
# ----------------------------------------------------------------------------

def _mix_np(z: np.ndarray) -> np.ndarray:
    z = (z ^ (z >> np.uint64(30))) * np.uint64(MUL1)
    z = (z ^ (z >> np.uint64(27))) * np.uint64(MUL2)
    return z ^ (z >> np.uint64(31))


def draws_np(seed: int, stream: int, start: int, count: int) -> np.ndarray:
    """Draws start .. start+count-1 of a stream as uint64."""
    s0 = np.uint64(stream_state(seed, stream))
    k = np.arange(start + 1, start + count + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        return _mix_np(s0 + k * np.uint64(GAMMA))


def _real_values_np(kind: str, prec: str, seed: int, stream: int, start: int, count: int):
    if kind == "uniform":
        d = draws_np(seed, stream, start, count)
        if prec == "f64":
            return (d >> np.uint64(11)).astype(np.float64) * 2.0 ** -52 - 1.0
        return ((d >> np.uint64(40)).astype(np.float32) * np.float32(2.0 ** -23)
                - np.float32(1.0))
    if kind == "normal":
        d = draws_np(seed, stream, 2 * start, 2 * count)
        u1 = ((d[0::2] >> np.uint64(11)).astype(np.float64) + 1.0) * 2.0 ** -53
        u2 = (d[1::2] >> np.uint64(11)).astype(np.float64) * 2.0 ** -53
        v = np.sqrt(-2.0 * np.log(u1)) * np.cos(2.0 * np.pi * u2)
        return v if prec == "f64" else v.astype(np.float32)
    raise ValueError(f"unknown value kind {kind!r}")


_NP_TYPES = {"f32": np.float32, "f64": np.float64,
             "c64": np.complex64, "c128": np.complex128}
_REAL_PREC = {"f32": "f32", "f64": "f64", "c64": "f32", "c128": "f64"}


def np_dtype(dtype: str):
    return _NP_TYPES[dtype]


def fill_np(out: np.ndarray, dtype: str, kind: str, seed: int, stream: int) -> np.ndarray:
    """Fill a flat numpy buffer with element values 0 .. out.size-1 of a stream."""
    flat = out.reshape(-1)
    n = flat.size
    prec = _REAL_PREC[dtype]
    cplx = dtype in ("c64", "c128")
    for s in range(0, n, _CHUNK):
        c = min(_CHUNK, n - s)
        if cplx:
            v = _real_values_np(kind, prec, seed, stream, 2 * s, 2 * c)
            flat[s:s + c].real = v[0::2]
            flat[s:s + c].imag = v[1::2]
        else:
            flat[s:s + c] = _real_values_np(kind, prec, seed, stream, s, c)
    return out


def values_np(dtype: str, kind: str, seed: int, stream: int, count: int) -> np.ndarray:
    out = np.empty(count, dtype=_NP_TYPES[dtype])
    return fill_np(out, dtype, kind, seed, stream)


# ----------------------------------------------------------------------------
# torch (any device); int64 arithmetic wraps modulo 2**64 like uint64
# ----------------------------------------------------------------------------

def _s64(x: int) -> int:
    x &= MASK64
    return x - (1 << 64) if x >> 63 else x


def _lsr(t, s: int):
    """Logical right shift of an int64 tensor holding uint64 bits."""
    return (t >> s) & ((1 << (64 - s)) - 1)


def _mix_torch(z):
    z = (z ^ _lsr(z, 30)) * _s64(MUL1)
    z = (z ^ _lsr(z, 27)) * _s64(MUL2)
    return z ^ _lsr(z, 31)


def draws_torch(seed: int, stream: int, start: int, count: int, device):
    import torch
    s0 = _s64(stream_state(seed, stream))
    k = torch.arange(start + 1, start + count + 1, dtype=torch.int64, device=device)
    return _mix_torch(k * _s64(GAMMA) + s0)


def _real_values_torch(kind, prec, seed, stream, start, count, device):
    import torch
    if kind == "uniform":
        d = draws_torch(seed, stream, start, count, device)
        if prec == "f64":
            return _lsr(d, 11).to(torch.float64) * 2.0 ** -52 - 1.0
        return _lsr(d, 40).to(torch.float32) * (2.0 ** -23) - 1.0
    if kind == "normal":
        d = draws_torch(seed, stream, 2 * start, 2 * count, device)
        u1 = (_lsr(d[0::2], 11).to(torch.float64) + 1.0) * 2.0 ** -53
        u2 = _lsr(d[1::2], 11).to(torch.float64) * 2.0 ** -53
        v = torch.sqrt(-2.0 * torch.log(u1)) * torch.cos(2.0 * np.pi * u2)
        return v if prec == "f64" else v.to(torch.float32)
    raise ValueError(f"unknown value kind {kind!r}")


def fill_torch(out, dtype: str, kind: str, seed: int, stream: int):
    """Fill a flat torch tensor (any device) with element values of a stream."""
    import torch
    flat = out.view(-1)
    n = flat.numel()
    prec = _REAL_PREC[dtype]
    cplx = dtype in ("c64", "c128")
    view = torch.view_as_real(flat) if cplx else flat
    for s in range(0, n, _CHUNK):
        c = min(_CHUNK, n - s)
        if cplx:
            v = _real_values_torch(kind, prec, seed, stream, 2 * s, 2 * c, out.device)
            view[s:s + c].copy_(v.view(c, 2))
        else:
            view[s:s + c].copy_(_real_values_torch(kind, prec, seed, stream, s, c,
                                                   out.device))
    return out


# ----------------------------------------------------------------------------
# small integer helpers for seeded layout choices
# ----------------------------------------------------------------------------

class IntStream:
    """Sequential integer draws from one stream (used for layout choices)."""

    def __init__(self, seed: int, stream: int):
        self.seed, self.stream, self.k = seed, stream, 0

    def next_u64(self) -> int:
        v = draw_int(self.seed, self.stream, self.k)
        self.k += 1
        return v

    def below(self, n: int) -> int:
        """Uniform integer in [0, n) by the multiply-high map (Lemire 2019)."""
        return (self.next_u64() * n) >> 64

    def between(self, lo: int, hi: int) -> int:
        """Uniform integer in [lo, hi]."""
        return lo + self.below(hi - lo + 1)

    def permutation(self, n: int) -> list[int]:
        """Fisher-Yates shuffle of range(n) (Knuth, TAOCP vol. 2, Alg. 3.4.2P)."""
        p = list(range(n))
        for i in range(n - 1, 0, -1):
            j = self.below(i + 1)
            p[i], p[j] = p[j], p[i]
        return p
