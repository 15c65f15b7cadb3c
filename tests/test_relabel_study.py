"""Greedy relabeling, grid-product volumes and the Sec. 7.2 study (host only)."""
import numpy as np
import pytest

import oracle
from workloads import gen
from workloads import layouts as L

costa = pytest.importorskip("paper_2106_06601_gb300")
from paper_2106_06601_gb300 import GridLayout, relabel_study  # noqa: E402


def _rand_V(P, seed, ties=False):
    rng = gen.IntStream(seed, 21)
    V = np.array([[rng.below(5 if ties else 10**6) for _ in range(P)] for _ in range(P)], np.int64)
    V[V % 3 == 0] = 0
    return V


@pytest.mark.parametrize("P", [1, 2, 3, 5, 8, 16, 31, 64, 100])
def test_greedy_matches_oracle_and_bound(P):
    for s in range(8):
        V = _rand_V(P, 50 * P + s, ties=(s % 2 == 1))
        sig, lv = costa.costa_relabel_greedy(V)
        osum, osig = oracle.lap_greedy(V)
        assert sig.tolist() == osig.tolist() and lv == osum
        assert sorted(sig.tolist()) == list(range(P))
        best = oracle.lap_optimum(V)
        assert 2 * lv >= best and lv <= best


def _spec_of_grid(g: GridLayout, P: int):
    """The same layout as a LayoutSpec with explicit owners (for the oracle)."""
    owner = g.grid[np.ix_(g.rp, g.cp)].astype(np.int32)
    return L.packed_blocks(g.rs, g.cs, owner, P)


@pytest.mark.parametrize("case", range(30))
def test_volume_grid_matches_element_count(case):
    rng = gen.IntStream(7, 300 + case)
    m, n = rng.between(1, 90), rng.between(1, 90)
    op = "NTC"[rng.below(3)]
    pr, pc = rng.between(1, 4), rng.between(1, 4)
    P = pr * pc
    bm, bn = (m, n) if op == "N" else (n, m)

    def rand_grid(mm, nn, rr, cc):
        if rng.below(2):
            return GridLayout.block_cyclic(mm, nn, rng.between(1, 12), rng.between(1, 12), rr, cc,
                                           "RC"[rng.below(2)], rng.permutation(rr * cc))
        rs = np.unique(np.concatenate([[0, mm], [rng.between(0, mm) for _ in range(5)]]))
        cs = np.unique(np.concatenate([[0, nn], [rng.between(0, nn) for _ in range(5)]]))
        return GridLayout(rs, [rng.below(rr) for _ in range(len(rs) - 1)], cs,
                          [rng.below(cc) for _ in range(len(cs) - 1)],
                          np.array(rng.permutation(rr * cc)).reshape(rr, cc))

    A = rand_grid(m, n, pr, pc)
    B = rand_grid(bm, bn, pr, pc)
    V = costa.costa_volume_grid(A, B, op, P)
    want = oracle.volume(op, _spec_of_grid(A, P), _spec_of_grid(B, P), P)
    assert np.array_equal(V, want)


def test_volume_grid_rejects_bad_input():
    A = GridLayout.block_cyclic(10, 10, 3, 3, 2, 2)
    B = GridLayout.block_cyclic(10, 11, 3, 3, 2, 2)
    with pytest.raises(costa.CostaError) as e:
        costa.costa_volume_grid(A, B, "N", 4)
    assert e.value.status == 3
    with pytest.raises(costa.CostaError) as e:
        costa.costa_volume_grid(A, A, "N", 2)          # grid ranks >= P
    assert e.value.status == 2


def test_study_endpoint_equal_blocks_is_100_percent():
    """Sec. 7.2: equal block sizes differ only by the rank numbering, and
    relabeling removes all remote volume (the figure's red dot)."""
    r = relabel_study.study_point(100000, 10, 10000, 10000)
    assert r["total"] == 10**10
    assert r["remote_identity"] > 0
    assert r["remote_optimal"] == 0 and r["reduction_optimal_pct"] == 100.0
    assert r["remote_greedy"] == 0


def test_study_curve_properties():
    rows = relabel_study.run(n=100000, grid=10, tgt_block=10000,
                             sizes=[1, 7, 100, 1000, 3333, 10000])
    for r in rows:
        assert r["total"] == 10**10
        assert 0 <= r["remote_optimal"] <= r["remote_greedy"] <= r["remote_identity"]
        assert 0.0 <= r["reduction_optimal_pct"] <= 100.0
    # block size 1 interleaves everything: the volume matrix is uniform and
    # no relabeling can help
    assert rows[0]["reduction_optimal_pct"] == pytest.approx(0.0, abs=1e-9)


def test_study_small_instance_against_oracle():
    """A scaled-down study point: the grid volumes equal the oracle's element
    count and the relabeled optimum equals brute force (P = 4)."""
    B = GridLayout.block_cyclic(60, 60, 7, 7, 2, 2, "R")
    A = GridLayout.block_cyclic(60, 60, 30, 30, 2, 2, "C")
    V = costa.costa_volume_grid(A, B, "N", 4)
    assert np.array_equal(V, oracle.volume("N", _spec_of_grid(A, 4), _spec_of_grid(B, 4), 4))
    _, best = costa.costa_relabel(V)
    assert best == oracle.lap_bruteforce(V)[0]


@pytest.mark.parametrize("order", ["R", "C"])
def test_grid_block_cyclic_matches_layout_owners(order):
    """costa_grid_block_cyclic's grid gives, block by block, the owners of the
    ScaLAPACK block-cyclic layout built independently in workloads.layouts."""
    rng = gen.IntStream(9, 77)
    for _ in range(20):
        m, n = rng.between(1, 300), rng.between(1, 300)
        mb, nb = rng.between(1, 40), rng.between(1, 40)
        pr, pc = rng.between(1, 5), rng.between(1, 5)
        perm = rng.permutation(pr * pc)
        g = GridLayout.block_cyclic(m, n, mb, nb, pr, pc, order, perm)
        spec = L.block_cyclic(m, n, mb, nb, pr, pc, grid_order=order, rank_perm=perm)
        assert np.array_equal(g.rs, spec.rsplit) and np.array_equal(g.cs, spec.csplit)
        assert np.array_equal(g.grid[np.ix_(g.rp, g.cp)], spec.owner)
