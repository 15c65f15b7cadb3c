"""The process-relabeling study of Sec. 7.2, computed through the library.

A 10^5 x 10^5 matrix is redistributed between two block-cyclic layouts on a
10 x 10 process grid: row-major grid numbering initially, column-major
finally; the target block size is fixed at 10^4 and the source block size
varies from 1 to 10^4.  For each source block size the volumes V come from
costa_volume_grid (1-D overlaps, no device work), and the remote volume
(volume whose sender is not its receiver) is compared without relabeling,
with the optimal relabeling (costa_relabel) and with the greedy one
(costa_relabel_greedy).  Reduction = (remote before - remote after) /
remote before, in percent.  The paper states that equal block sizes give a
reduction of 100%.

    python -m paper_2106_06601_gb300.relabel_study [--n 100000] [--grid 10]
"""
from __future__ import annotations

import argparse
import json

import numpy as np

from . import GridLayout, costa_relabel, costa_relabel_greedy, costa_volume_grid

DEFAULT_SIZES = [1, 2, 3, 5, 7, 10, 20, 33, 50, 100, 200, 333, 500, 1000, 2000, 2500, 3333,
                 5000, 7777, 9999, 10000]


def study_point(n: int, grid: int, src_block: int, tgt_block: int) -> dict:
    B = GridLayout.block_cyclic(n, n, src_block, src_block, grid, grid, "R")
    A = GridLayout.block_cyclic(n, n, tgt_block, tgt_block, grid, grid, "C")
    P = grid * grid
    V = costa_volume_grid(A, B, "N", P)
    total = int(V.sum())
    remote0 = total - int(np.trace(V))
    _, opt = costa_relabel(V)
    _, greedy = costa_relabel_greedy(V)
    red = lambda local: 100.0 * (remote0 - (total - local)) / remote0 if remote0 else 0.0
    return {"src_block": src_block, "tgt_block": tgt_block, "total": total,
            "remote_identity": remote0, "remote_optimal": total - opt,
            "remote_greedy": total - greedy, "reduction_optimal_pct": red(opt),
            "reduction_greedy_pct": red(greedy)}


def run(n: int = 100000, grid: int = 10, tgt_block: int = 10000, sizes=None) -> list[dict]:
    return [study_point(n, grid, b, tgt_block) for b in (sizes or DEFAULT_SIZES)]


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--n", type=int, default=100000)
    ap.add_argument("--grid", type=int, default=10)
    ap.add_argument("--target-block", type=int, default=10000)
    ap.add_argument("--json", action="store_true")
    a = ap.parse_args()
    rows = run(a.n, a.grid, a.target_block)
    if a.json:
        print(json.dumps(rows))
        return
    print(f"{'source block':>12} {'remote (identity)':>18} {'optimal':>14} {'greedy':>14} "
          f"{'reduction opt %':>15} {'greedy %':>9}")
    for r in rows:
        print(f"{r['src_block']:>12} {r['remote_identity']:>18} {r['remote_optimal']:>14} "
              f"{r['remote_greedy']:>14} {r['reduction_optimal_pct']:>15.2f} "
              f"{r['reduction_greedy_pct']:>9.2f}")


if __name__ == "__main__":
    main()
