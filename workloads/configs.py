"""Seeded synthetic problems shaped like the paper's workloads.

Each problem is one instance of A = alpha * op(B) + beta * A (Eq. 1 of Sec. 5)
between a source layout L(B) and a target layout L(A):

  c1  256 x 256 f64, B block-cyclic 16x16 on a 2x2 row-major grid -> A block-cyclic
      32x32 on a 2x2 column-major grid; op = N, alpha = 1, beta = 0; P = 4.
  c2  8192 x 8192 f64, B block-cyclic 64x64 on 4x4 -> A block-cyclic 128x128 on 4x4
      with a seeded random rank permutation; op = T, alpha = 2, beta = 0.5; P = 16.
      (Stands in for the Sec. 7.1 ScaLAPACK reshuffle/transpose, 32 -> 128 blocks.)
  c3  16384 x 16384 c128, B block-cyclic 32x32 on 8x8 -> A irregular 8x8 grid
      (seeded splits, block sizes 512..3584) with seeded owners; op = C, alpha = 1,
      beta = 0; P = 64.
  c4  64 independent 2048 x 3072 f32 pairs, each side block-cyclic on a 4x4 grid
      with block sizes drawn from {16, 32, 64, 128}; op = N for even, T for odd
      instances; alpha = 1, beta = 0; P = 16; one batched call (Sec. 6).
  c5  RPA-like tall-skinny: B 131072 x 4096 f64 normal(0,1), block-cyclic 32x32
      on a 16x16 grid -> A 4096 x 131072 in 256 row panels of 16 rows, rank k owns
      panel k; op = T, alpha = 1, beta = 1; P = 256.  (Stands in for the
      Sec. 7.3 RPA matrices, 3,473,408 x 17,408, scaled down.)

Value seeds: problem set k uses seed 2106066010 + k.  Buffer r of the source of
instance t draws from stream SRC + 4096 t + r; of the target, TGT + 4096 t + r.
Layout choices (permutations, splits, block sizes) draw from stream LAYOUT + t.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

from . import layouts as L
from .gen import IntStream

SEED0 = 2106066010
SRC, TGT, LAYOUT = 1 << 20, 2 << 20, 3 << 20


@dataclass
class Problem:
    name: str
    dtype: str            # "f32" | "f64" | "c64" | "c128"
    op: str               # "N" | "T" | "C"
    alpha: complex
    beta: complex
    A: L.LayoutSpec       # target
    B: L.LayoutSpec       # source
    b_kind: str = "uniform"   # value distribution of B
    a_kind: str = "uniform"   # prefill of A: "uniform" | "normal" | "nan"
    seed: int = SEED0
    index: int = 0        # instance index inside a batch (selects value streams)
    relabel: bool = True

    def src_stream(self, r: int) -> int:
        return SRC + 4096 * self.index + r

    def tgt_stream(self, r: int) -> int:
        return TGT + 4096 * self.index + r

    @property
    def esize(self) -> int:
        return {"f32": 4, "f64": 8, "c64": 8, "c128": 16}[self.dtype]

    def algorithmic_bytes(self) -> int:
        """Read B + read A (only if beta != 0) + write A."""
        n = self.A.m * self.A.n
        return n * self.esize * (3 if self.beta != 0 else 2)


def _seed(k: int) -> int:
    return SEED0 + k


def c1() -> Problem:
    B = L.block_cyclic(256, 256, 16, 16, 2, 2, grid_order="R", name="B")
    A = L.block_cyclic(256, 256, 32, 32, 2, 2, grid_order="C", name="A")
    return Problem("c1", "f64", "N", 1.0, 0.0, A, B, "uniform", "nan", _seed(1))


def c2(n: int = 8192) -> Problem:
    perm = IntStream(_seed(2), LAYOUT).permutation(16)
    B = L.block_cyclic(n, n, 64, 64, 4, 4, grid_order="R", name="B")
    A = L.block_cyclic(n, n, 128, 128, 4, 4, grid_order="R", rank_perm=perm, name="A")
    return Problem("c2", "f64", "T", 2.0, 0.5, A, B, "uniform", "uniform", _seed(2))


def c3(n: int = 16384) -> Problem:
    rng = IntStream(_seed(3), LAYOUT)
    scale = n / 16384
    lo, hi = max(1, int(512 * scale)), max(1, int(3584 * scale))
    rs = L.random_splits(n, 8, lo, hi, rng)
    cs = L.random_splits(n, 8, lo, hi, rng)
    owner = np.array(rng.permutation(64), dtype=np.int32).reshape(8, 8)
    B = L.block_cyclic(n, n, 32, 32, 8, 8, grid_order="R", name="B")
    A = L.packed_blocks(rs, cs, owner, 64, name="A")
    return Problem("c3", "c128", "C", 1.0, 0.0, A, B, "uniform", "nan", _seed(3))


def c4(count: int = 64, m: int = 2048, n: int = 3072) -> list[Problem]:
    sizes = (16, 32, 64, 128)
    out = []
    for t in range(count):
        rng = IntStream(_seed(4), LAYOUT + t)
        mbB, nbB, mbA, nbA = (sizes[rng.below(4)] for _ in range(4))
        op = "N" if t % 2 == 0 else "T"
        B = L.block_cyclic(m, n, mbB, nbB, 4, 4, grid_order="R", name=f"B{t}")
        am, an = (m, n) if op == "N" else (n, m)
        A = L.block_cyclic(am, an, mbA, nbA, 4, 4, grid_order="R", name=f"A{t}")
        out.append(Problem(f"c4[{t}]", "f32", op, 1.0, 0.0, A, B, "uniform", "nan",
                           _seed(4), index=t))
    return out


def c5(rows: int = 131072, cols: int = 4096) -> Problem:
    B = L.block_cyclic(rows, cols, 32, 32, 16, 16, grid_order="R", name="B")
    A = L.row_panels(cols, rows, 256, name="A")
    return Problem("c5", "f64", "T", 1.0, 1.0, A, B, "normal", "normal", _seed(5))


CONFIGS = {"c1": c1, "c2": c2, "c3": c3, "c4": c4, "c5": c5}


def small_blocks(n: int = 8192, mb: int = 8, dtype: str = "f64") -> Problem:
    """The small-block case (not one of the configurations above): c2's
    shape and scalars with mb x mb blocks on both sides, 4 x 4 grids, the
    target's owners a seeded permutation."""
    perm = IntStream(_seed(6), LAYOUT).permutation(16)
    B = L.block_cyclic(n, n, mb, mb, 4, 4, grid_order="R", name="B")
    A = L.block_cyclic(n, n, mb, mb, 4, 4, grid_order="R", rank_perm=perm, name="A")
    return Problem(f"bc{mb}", dtype, "T", 2.0, 0.5, A, B, "uniform", "uniform", _seed(6))


def c5b(rows: int = 131072, cols: int = 4096) -> Problem:
    """The other reading of c5's target: A (cols x rows) in 256 column panels
    of rows / 256 columns, rank k owning panel k, column-major with ld = cols
    (each panel one contiguous buffer)."""
    B = L.block_cyclic(rows, cols, 32, 32, 16, 16, grid_order="R", name="B")
    w = rows // 256
    A = L.packed_blocks([0, cols], [k * w for k in range(257)], np.arange(256, dtype=np.int32).reshape(1, 256),
                        256, name="A")
    return Problem("c5b", "f64", "T", 1.0, 1.0, A, B, "normal", "normal", _seed(5))


# Further workloads for measurement only.
def c2_general_beta(n: int = 8192) -> Problem:
    """c2's layouts and op with a general beta (alpha = -0.3, beta = 0.7):
    the combine kind whose source tiles are staged by TMA (not one of the
    configurations above)."""
    p = c2(n)
    p.name = "c2g"
    p.alpha, p.beta = -0.3, 0.7
    return p


def f32_lld(n: int = 8192, pad: int = 1) -> Problem:
    """A ScaLAPACK-style target with an odd local leading dimension: f32,
    T copy, B BC64 4x4 -> A BC128 4x4 with A's ld = local rows + pad (pad =
    1: ld = 1 mod 4, every target run off 16-byte boundaries; pad = 0: the
    same layouts aligned).  Not a configuration."""
    B = L.block_cyclic(n, n, 64, 64, 4, 4, name="B")
    A = L.block_cyclic(n, n, 128, 128, 4, 4, ld_pad=pad, name="A")
    return Problem("ld1" if pad else "ld0", "f32", "T", 1.0, 0.0, A, B, "uniform", "nan", _seed(7))


def odd_blocks(n: int = 8192, dtype: str = "f64") -> Problem:
    """Odd block sizes on both sides: T copy, B BC50 4x4 -> A BC75 4x4 (cells
    of 25 x 25 and 25 x 50 elements, runs at odd 8-byte phases).  Not a
    configuration."""
    B = L.block_cyclic(n, n, 50, 50, 4, 4, name="B")
    A = L.block_cyclic(n, n, 75, 75, 4, 4, name="A")
    return Problem("odd", dtype, "T", 1.0, 0.0, A, B, "uniform", "nan", _seed(7))


def c2_complex_scalars(n: int = 8192, complex_beta: bool = True) -> Problem:
    """c2's layouts and op with double complex data and complex scalars:
    alpha = 1, beta = 0.5 + 0.25i (every component a sum of four products)
    or alpha = 0.3 - 0.4i, beta = 0 (two products; A is not read).  The
    kinds whose arithmetic, not memory, sets the rate.  Not configurations."""
    p = c2(n)
    p.dtype = "c128"
    if complex_beta:
        p.name, p.alpha, p.beta = "zb", 1.0, complex(0.5, 0.25)
    else:
        p.name, p.alpha, p.beta, p.a_kind = "za", complex(0.3, -0.4), 0.0, "nan"
    return p


EXTRA_WORKLOADS = {"bc8": small_blocks, "c5b": c5b, "c2g": c2_general_beta,
                   "ld1": f32_lld, "ld0": lambda: f32_lld(pad=0), "odd": odd_blocks,
                   "zb": c2_complex_scalars, "za": lambda: c2_complex_scalars(complex_beta=False)}

# The same layouts and tile shapes at about 1 GB on the device, for profiler
# captures (the workloads proper stay the ones above).
CONFIGS_SMALL = {"c1": c1, "c2": lambda: c2(4096), "c3": lambda: c3(8192),
                 "c4": lambda: c4(16), "c5": lambda: c5(rows=16384), "bc8": lambda: small_blocks(4096),
                 "c2g": lambda: c2_general_beta(4096),
                 "ld1": lambda: f32_lld(8192), "ld0": lambda: f32_lld(8192, 0), "odd": lambda: odd_blocks(4096),
                 "c5b": lambda: c5b(rows=16384), "zb": lambda: c2_complex_scalars(4096),
                 "za": lambda: c2_complex_scalars(4096, complex_beta=False)}

WORKLOAD_TEXT = {
    "c1": "256x256 f64 BC16 2x2R -> BC32 2x2C, N, alpha=1 beta=0, P=4",
    "c2": "8192x8192 f64 BC64 4x4 -> BC128 4x4 permuted owners, T, alpha=2 beta=0.5, P=16",
    "c3": "16384x16384 c128 BC32 8x8 -> irregular 8x8 (512..3584), C, alpha=1 beta=0, P=64",
    "c4": "64 x 2048x3072 f32 BC{16..128} 4x4, N/T alternating, alpha=1 beta=0, P=16, batched",
    "c5": "131072x4096 f64 BC32 16x16 -> 4096x131072 in 256 row panels, T, alpha=1 beta=1, P=256",
    "bc8": "8192x8192 f64 BC8 4x4 -> BC8 4x4 permuted owners, T, alpha=2 beta=0.5, P=16 "
           "(small-block case, not a configuration)",
    "c5b": "131072x4096 f64 BC32 16x16 -> 4096x131072 in 256 column panels of 512, T, alpha=1 beta=1, "
           "P=256 (the other reading of c5's target)",
    "c2g": "8192x8192 f64 BC64 4x4 -> BC128 4x4 permuted owners, T, alpha=-0.3 beta=0.7, P=16 "
           "(c2 with a general beta: TMA-staged source tiles; not a configuration)",
    "ld1": "8192x8192 f32 BC64 4x4 -> BC128 4x4 with A's ld = 1 mod 4, T, alpha=1 beta=0, P=16 "
           "(misaligned target runs; not a configuration)",
    "ld0": "8192x8192 f32 BC64 4x4 -> BC128 4x4, T, alpha=1 beta=0, P=16 (ld1's layouts aligned; "
           "not a configuration)",
    "odd": "8192x8192 f64 BC50 4x4 -> BC75 4x4, T, alpha=1 beta=0, P=16 (odd block sizes; "
           "not a configuration)",
    "zb": "8192x8192 c128 BC64 4x4 -> BC128 4x4 permuted owners, T, alpha=1 beta=0.5+0.25i, P=16 "
          "(complex beta: four products per component; not a configuration)",
    "za": "8192x8192 c128 BC64 4x4 -> BC128 4x4 permuted owners, T, alpha=0.3-0.4i beta=0, P=16 "
          "(complex alpha: two products per component; not a configuration)",
}


# ----------------------------------------------------------------------------
# randomized small problems for parity fuzzing
# ----------------------------------------------------------------------------

def _rand_splits(extent: int, rng: IntStream, allow_empty: bool) -> np.ndarray:
    cuts = [0]
    while cuts[-1] < extent:
        step = rng.between(0 if allow_empty and rng.below(6) == 0 else 1,
                           max(1, min(extent, 1 + rng.below(48))))
        cuts.append(min(extent, cuts[-1] + step))
    if extent == 0:
        cuts = [0]
    return np.array(cuts, dtype=np.int64)


def _rand_layout(m: int, n: int, P: int, rng: IntStream, name: str) -> L.LayoutSpec:
    kind = rng.below(3)
    if kind == 0 and m > 0 and n > 0:
        # block-cyclic on a random grid whose size divides into P ranks
        pr = [d for d in range(1, P + 1) if P % d == 0][rng.below(
            len([d for d in range(1, P + 1) if P % d == 0]))]
        pc = P // pr
        perm = rng.permutation(P) if rng.below(2) else None
        return L.block_cyclic(m, n, rng.between(1, 40), rng.between(1, 40), pr, pc,
                              grid_order="RC"[rng.below(2)], rank_perm=perm,
                              storage="CR"[rng.below(2)], ld_pad=rng.below(3) * rng.below(5),
                              name=name)
    rs = _rand_splits(m, rng, allow_empty=True)
    cs = _rand_splits(n, rng, allow_empty=True)
    nbr, nbc = len(rs) - 1, len(cs) - 1
    owner = np.array([[rng.below(P) for _ in range(nbc)] for _ in range(nbr)],
                     dtype=np.int32).reshape(nbr, nbc)
    order = np.array([[rng.below(2) for _ in range(nbc)] for _ in range(nbr)],
                     dtype=np.int32).reshape(nbr, nbc)
    pad = np.array([[rng.below(3) * rng.below(4) for _ in range(nbc)] for _ in range(nbr)],
                   dtype=np.int64).reshape(nbr, nbc)
    return L.packed_blocks(rs, cs, owner, P, order=order, ld_pad=pad, name=name)


SCALARS = [(1.0, 0.0), (2.0, 0.5), (1.0, 1.0), (0.5, -1.25), (-0.3, 0.7), (1.5, 0.0)]
COMPLEX_SCALARS = [(complex(0.5, -0.75), complex(1.0, 0.0)),
                   (complex(1.0, 0.0), complex(0.25, 2.0)),
                   (complex(-0.6, 0.3), 0.0)]


SMALL_BLOCKS = (1, 2, 3, 4, 5, 8, 12, 16, 24)
ALIGNED_SMALL_BLOCKS = (4, 8, 12, 16)


def small_block_problem(case: int) -> Problem:
    """Block-cyclic layouts with small blocks on 2 x 2 grids, both storage
    orders, cycling through the element types and ops; drawn from stream
    LAYOUT + 5000 + case.  Odd cases take odd block sizes (1 .. 24) and padded
    leading dimensions; even cases take block sizes that are multiples of 4,
    matrix sizes that are multiples of 16 and unpadded storage, so that their
    tiles start on 16-byte boundaries."""
    rng = IntStream(SEED0 + 200, LAYOUT + 5000 + case)
    dtype = ("f32", "f64", "c64", "c128")[(case // 2) % 4]
    op = "NTC"[(case // 8) % 3]
    aligned = case % 2 == 0
    if aligned:
        m, n = 16 * rng.between(1, 6), 16 * rng.between(1, 6)
        sizes, pad = ALIGNED_SMALL_BLOCKS, lambda: 0
    else:
        m, n = rng.between(1, 90), rng.between(1, 90)
        sizes, pad = SMALL_BLOCKS, lambda: rng.below(3)
    mbB, nbB, mbA, nbA = (sizes[rng.below(len(sizes))] for _ in range(4))
    sb, sa = ("C", "R")[(case // 24) % 2], ("C", "R")[(case // 48) % 2]
    B = L.block_cyclic(m, n, mbB, nbB, 2, 2, storage=sb, ld_pad=pad(), name="B")
    am, an = (m, n) if op == "N" else (n, m)
    A = L.block_cyclic(am, an, mbA, nbA, 2, 2, grid_order="C", storage=sa, ld_pad=pad(), name="A")
    alpha, beta = SCALARS[rng.below(len(SCALARS))]
    a_kind = "nan" if beta == 0 else "uniform"
    return Problem(f"small{case}", dtype, op, alpha, beta, A, B, "uniform", a_kind, SEED0 + 200,
                   index=case % 64)


def fuzz_problem(case: int, *, dtype=None, op=None, P=None, max_dim: int = 160) -> Problem:
    """A random small problem; everything is drawn from stream LAYOUT + case."""
    rng = IntStream(SEED0 + 100, LAYOUT + case)
    dtype = dtype or ("f32", "f64", "c64", "c128")[rng.below(4)]
    op = op or "NTC"[rng.below(3)]
    P = P or (1, 2, 3, 4, 7, 8)[rng.below(6)]
    m = rng.between(1, max_dim)
    n = rng.between(1, max_dim)
    B = _rand_layout(m, n, P, rng, "B")
    am, an = (m, n) if op == "N" else (n, m)
    A = _rand_layout(am, an, P, rng, "A")
    if dtype in ("c64", "c128") and rng.below(3) == 0:
        alpha, beta = COMPLEX_SCALARS[rng.below(len(COMPLEX_SCALARS))]
    else:
        alpha, beta = SCALARS[rng.below(len(SCALARS))]
    a_kind = "nan" if beta == 0 else "uniform"
    return Problem(f"fuzz{case}", dtype, op, alpha, beta, A, B, "uniform", a_kind,
                   SEED0 + 100, index=case % 64)
