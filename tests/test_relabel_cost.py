"""Relabeling under the topology cost of Sec. 3 (w = L + B * V for remote
packages), against brute force over W(G_sigma) computed from its definition
(Def. RG, Eq. WG), Lemma 1, and the reduction to the volume-only case."""
import numpy as np
import pytest

import oracle
from workloads import gen

costa = pytest.importorskip("paper_2106_06601_gb300")


def _problem(P, seed):
    rng = gen.IntStream(seed, 31)
    V = np.array([[rng.below(1000) for _ in range(P)] for _ in range(P)], np.int64)
    V[V % 4 == 0] = 0
    # a two-level topology: cheap inside groups of 2 ranks, expensive across
    lat = np.zeros((P, P))
    bw = np.zeros((P, P))
    for i in range(P):
        for j in range(P):
            if i != j:
                same = i // 2 == j // 2
                lat[i, j] = (1.0 if same else 20.0) + rng.below(3)
                bw[i, j] = (0.5 if same else 2.0) + rng.below(100) / 100.0
    return V, lat, bw


@pytest.mark.parametrize("P", [1, 2, 3, 4, 5, 6, 7, 8])
def test_cost_relabel_equals_bruteforce(P):
    for s in range(6):
        V, lat, bw = _problem(P, 100 * P + s)
        sigma, c0, c1 = costa.costa_relabel_cost(V, lat, bw)
        assert sorted(sigma.tolist()) == list(range(P))
        best, _ = oracle.copr_bruteforce_cost(V, lat, bw)
        w = oracle.cost_W(V, lat, bw, sigma)
        assert w == pytest.approx(best, rel=1e-12, abs=1e-9)
        assert c1 == pytest.approx(w, rel=1e-12, abs=1e-9)
        assert c0 == pytest.approx(oracle.cost_W(V, lat, bw, np.arange(P)), rel=1e-12, abs=1e-9)


def test_lemma1_with_topology_cost():
    """Total gain sum_j delta(j, sigma(j)) (Eq. delta, with N_L(p_x) the
    senders of non-empty packages to x) equals W(G) - W(G_sigma)."""
    P = 6
    V, lat, bw = _problem(P, 7)

    def w(i, j, v):
        return 0.0 if (v == 0 or i == j) else lat[i, j] + bw[i, j] * v

    ident = np.arange(P)
    for s in range(10):
        sig = np.array(gen.IntStream(s, 41).permutation(P))
        gain = sum(w(i, x, V[i, x]) - w(i, sig[x], V[i, x])
                   for x in range(P) for i in range(P) if V[i, x] > 0)
        lhs = oracle.cost_W(V, lat, bw, ident) - oracle.cost_W(V, lat, bw, sig)
        assert gain == pytest.approx(lhs, rel=1e-12, abs=1e-9)


def test_volume_cost_reduces_to_relabel():
    """lat = 0 and bw = 1 off the diagonal is the locally-free volume cost
    (Eq. 2): minimizing W is maximizing the local volume."""
    P = 12
    rng = gen.IntStream(3, 51)
    V = np.array([[rng.below(100) for _ in range(P)] for _ in range(P)], np.int64)
    lat = np.zeros((P, P))
    bw = np.ones((P, P)) - np.eye(P)
    sigma, _, c1 = costa.costa_relabel_cost(V, lat, bw)
    _, local = costa.costa_relabel(V)
    assert c1 == pytest.approx(V.sum() - local)
    assert oracle.objective(V, sigma) == local


def test_cost_relabel_rejects_bad_input():
    V = np.zeros((2, 2), np.int64)
    with pytest.raises(costa.CostaError):
        costa.costa_relabel_cost(V, np.full((2, 2), np.nan), np.zeros((2, 2)))
    with pytest.raises(costa.CostaError):
        costa.costa_relabel_cost(-np.ones((2, 2), np.int64), np.zeros((2, 2)), np.zeros((2, 2)))
