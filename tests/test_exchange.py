"""The multi-GPU exchange's host-side plan (Sec. 6 "Implementation", Alg. 3),
on the CPU: the partition of the tiles between G processes, the per-pair
volumes, package sizes and offsets, and, through a numpy emulation of the
three tile lists, the final A against the oracle.  The exchange itself runs
as an in-process copy of the segments and as a world_size-2 gloo
all_to_all_single.  Relabeling for a placement is checked against brute force
over W(G_sigma)."""
import dataclasses
import os
import socket

import numpy as np
import pytest

import oracle
from tests._exchange import aligned_bytes, apply_list, block_placement, host_ptrs
from workloads import configs as C
from workloads.materialize import host_problem

costa = pytest.importorskip("paper_2106_06601_gb300")

SCALARS = [(1.0, 0.0), (2.0, 0.5), (-0.5, 0.0)]


def _problem(case, dtype=None, op=None, P=None):
    p = C.fuzz_problem(case, dtype=dtype, op=op, P=P)
    p.alpha, p.beta = SCALARS[case % len(SCALARS)]
    p.a_kind = "nan" if p.beta == 0 else "uniform"
    return p


def _placement(P, G, case):
    if case % 2 == 0:
        return block_placement(P, G)
    rng = np.random.default_rng(case)
    return rng.integers(0, G, P).astype(np.int32)


def _layouts(p, Bh, Ah, place, g):
    LA = costa.costa_layout_from_spec(p.A, p.dtype, host_ptrs(p.A, Ah, place, g))
    LB = costa.costa_layout_from_spec(p.B, p.dtype, host_ptrs(p.B, Bh, place, g))
    return LA, LB


def _check_plan(p, G, place, g, LA, LB, sb, rb, V):
    """Package sizes, volumes and offsets of process g's lists."""
    es = np.dtype(Bh_dtype(p.dtype)).itemsize
    send = aligned_bytes(int(sb.sum()))
    recv = aligned_bytes(int(rb.sum()))
    s0, r0 = send.ctypes.data, recv.ctypes.data
    pack, vol = costa.costa_debug_exchange(LA, LB, p.op, G, place, g, s0, r0, "pack")
    local, _ = costa.costa_debug_exchange(LA, LB, p.op, G, place, g, s0, r0, "local")
    unpack, _ = costa.costa_debug_exchange(LA, LB, p.op, G, place, g, s0, r0, "unpack")
    pl = np.asarray(place)
    on = [pl == h for h in range(G)]
    for h in range(G):
        assert vol[0, h] == (0 if h == g else V[np.ix_(on[g], on[h])].sum())
        assert vol[1, h] == (0 if h == g else V[np.ix_(on[h], on[g])].sum())
    assert (local["nx"].astype(np.int64) * local["ny"]).sum() == V[np.ix_(on[g], on[g])].sum()
    # packed tiles fill each send segment back to back, in order, 16-byte aligned
    displ = np.concatenate([[0], np.cumsum(sb)[:-1]])
    pos = s0 + displ.copy()
    seg = np.searchsorted(np.cumsum(sb), pack["dst"].astype(np.int64) - s0, side="right")
    for d, h in zip(pack, seg):
        assert int(d["dst"]) == pos[h] and int(d["dst"]) % 16 == 0
        pos[h] += int(d["dld"]) * int(d["ny"]) * es
    assert np.array_equal(pos - s0, displ + sb)
    return send, recv, pack, local, unpack


def Bh_dtype(dtype):
    return {"f32": np.float32, "f64": np.float64, "c64": np.complex64, "c128": np.complex128}[dtype]


@pytest.mark.parametrize("case", range(24))
def test_exchange_in_process(case):
    """G processes emulated in one process over shared host arenas: every
    process packs, the segments are copied to their receivers, every process
    runs its local and unpack lists; A equals the oracle's result."""
    p = _problem(case)
    P = p.A.nranks
    G = (1, 2, 3, 4)[case % 4]
    place = _placement(P, G, case)
    Bh, Ah = host_problem(p)
    want = Ah.copy()
    oracle.transform(p.dtype, p.op, p.alpha, p.beta, p.A, want.buffers(), p.B, Bh.buffers())
    V = oracle.volume(p.op, p.A, p.B, P)
    procs = []
    for g in range(G):
        LA, LB = _layouts(p, Bh, Ah, place, g)
        sb, rb = costa.costa_exchange_sizes(LA, LB, p.op, G, place, g)
        procs.append((LA, LB, sb, rb) + _check_plan(p, G, place, g, LA, LB, sb, rb, V))
    for g in range(G):  # send[g -> h] is recv[h <- g]
        for h in range(G):
            assert procs[g][2][h] == procs[h][3][g]
    for (LA, LB, sb, rb, send, recv, pack, local, unpack) in procs:
        apply_list(pack, p.dtype, copy=True)
    for g in range(G):
        recv = procs[g][5]
        rdispl = np.concatenate([[0], np.cumsum(procs[g][3])[:-1]])
        for h in range(G):
            sdispl = np.concatenate([[0], np.cumsum(procs[h][2])[:-1]])
            n = int(procs[g][3][h])
            recv[rdispl[h]:rdispl[h] + n] = procs[h][4][sdispl[g]:sdispl[g] + n]
    for (LA, LB, sb, rb, send, recv, pack, local, unpack) in procs:
        apply_list(local, p.dtype, p.alpha, p.beta)
        apply_list(unpack, p.dtype, p.alpha, p.beta)
    ok = (Ah.arena == want.arena) | (np.isnan(Ah.arena) & np.isnan(want.arena))
    assert ok.all(), f"{(~ok).sum()} elements differ"
    for pr in procs:
        pr[0].destroy()
        pr[1].destroy()


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _gloo_worker(rank, world, port, case, q):
    import torch
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import paper_2106_06601_gb300 as cst
        p = _problem(case, P=8)
        P, G, g = p.A.nranks, world, rank
        place = block_placement(P, G)
        Bh, Ah = host_problem(p)       # this process's own copy of both matrices
        LA = cst.costa_layout_from_spec(p.A, p.dtype, host_ptrs(p.A, Ah, place, g))
        LB = cst.costa_layout_from_spec(p.B, p.dtype, host_ptrs(p.B, Bh, place, g))
        sb, rb = cst.costa_exchange_sizes(LA, LB, p.op, G, place, g)
        # every process's counts, to check that sends and receives pair up
        allc = [torch.zeros(2 * G, dtype=torch.int64) for _ in range(G)]
        dist.all_gather(allc, torch.from_numpy(np.concatenate([sb, rb])))
        allc = torch.stack(allc).numpy()
        assert all(allc[a, b] == allc[b, G + a] for a in range(G) for b in range(G))
        send, recv = aligned_bytes(int(sb.sum())), aligned_bytes(int(rb.sum()))
        lists = {w: cst.costa_debug_exchange(LA, LB, p.op, G, place, g, send.ctypes.data,
                                             recv.ctypes.data, w)[0]
                 for w in ("pack", "local", "unpack")}
        apply_list(lists["pack"], p.dtype, copy=True)
        dist.all_to_all_single(torch.from_numpy(recv), torch.from_numpy(send),
                               rb.tolist(), sb.tolist())
        apply_list(lists["local"], p.dtype, p.alpha, p.beta)
        apply_list(lists["unpack"], p.dtype, p.alpha, p.beta)
        Bw, Aw = host_problem(p)
        oracle.transform(p.dtype, p.op, p.alpha, p.beta, p.A, Aw.buffers(), p.B, Bw.buffers())
        # this process's blocks hold the oracle's result; the others are untouched
        _, A0 = host_problem(p)
        mine = np.zeros(Ah.arena.size, bool)
        for bi in range(p.A.nbr):
            for bj in range(p.A.nbc):
                if place[p.A.owner[bi, bj]] != g:
                    continue
                h = int(p.A.rsplit[bi + 1] - p.A.rsplit[bi])
                w = int(p.A.csplit[bj + 1] - p.A.csplit[bj])
                base = int(Ah.starts[p.A.buf[bi, bj]] + p.A.off[bi, bj])
                ld = int(p.A.ld[bi, bj])
                for r in range(h):
                    for c in range(w):
                        mine[base + (r + c * ld if p.A.order[bi, bj] == 0 else r * ld + c)] = True
        eq = lambda x, y: (x == y) | (np.isnan(x) & np.isnan(y))
        q.put((rank, bool(eq(Ah.arena[mine], Aw.arena[mine]).all()),
               bool(eq(Ah.arena[~mine], A0.arena[~mine]).all()), int(sb.sum()), int(rb.sum())))
        LA.destroy()
        LB.destroy()
    except Exception as e:  # reported to the parent
        q.put((rank, repr(e), None, 0, 0))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("case", [0, 1, 2, 5])
def test_exchange_gloo_world2(case):
    """Two processes, each with its own copy of the matrices and the ranks
    0-3 / 4-7: pack, gloo all_to_all_single of the segments, local, unpack."""
    torch = pytest.importorskip("torch")
    import torch.multiprocessing as mp
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_gloo_worker, args=(r, world, port, case, q)) for r in range(world)]
    for pr in procs:
        pr.start()
    out = sorted(q.get(timeout=240) for _ in range(world))
    for pr in procs:
        pr.join(timeout=60)
    for rank, mine_ok, rest_ok, nsend, nrecv in out:
        assert mine_ok is True, (rank, mine_ok)
        assert rest_ok is True, rank


@pytest.mark.parametrize("P", [2, 3, 4, 5, 6])
def test_relabel_placement_equals_bruteforce(P):
    """W(G_sigma) with packages kept on their process free, intra-GPU ones at
    intra * v and cross-GPU ones at v (Sec. 3 topology cost) is minimized:
    the optimum equals brute force over all permutations (Def. COPR)."""
    rng = np.random.default_rng(40 + P)
    for s in range(5):
        V = rng.integers(0, 50, (P, P)).astype(np.int64)
        V[V % 4 == 0] = 0
        G = 1 + s % min(3, P)
        place = rng.integers(0, G, P).astype(np.int32)
        intra = (0.0, 0.25, 1.0)[s % 3]
        sigma, c0, c1 = costa.costa_relabel_placement(V, G, place, intra)
        lat = np.zeros((P, P))
        bw = np.where(place[:, None] == place[None, :], intra, 1.0) * (1 - np.eye(P))
        best, _ = oracle.copr_bruteforce_cost(V, lat, bw)
        assert c1 == pytest.approx(best, abs=1e-9)
        assert oracle.cost_W(V, lat, bw, sigma) == pytest.approx(c1, abs=1e-9)
        assert c0 == pytest.approx(oracle.cost_W(V, lat, bw, np.arange(P)), abs=1e-9)


def test_relabeled_exchange_moves_the_optimal_volume():
    """With intra = 0, W(G_sigma) is the volume that crosses GPUs.  A's layout
    with its owners relabeled (label q to process sigma(q)) gives an exchange
    whose cross-GPU volume is exactly that, and the emulated result still
    equals the oracle's."""
    p = _problem(7, dtype="f64", op="T", P=8)
    P, G = 8, 2
    place = block_placement(P, G)
    V = oracle.volume(p.op, p.A, p.B, P)
    sigma, c0, c1 = costa.costa_relabel_placement(V, G, place, 0.0)
    # label q's blocks now belong to process sigma(q); their storage is unchanged
    p.A = dataclasses.replace(p.A, owner=sigma[p.A.owner].astype(np.int32))
    Bh, Ah = host_problem(p)
    want = Ah.copy()
    oracle.transform(p.dtype, p.op, p.alpha, p.beta, p.A, want.buffers(), p.B, Bh.buffers())
    cross = 0
    for g in range(G):
        LA, LB = _layouts(p, Bh, Ah, place, g)
        _, vol = costa.costa_debug_exchange(LA, LB, p.op, G, place, g, 0, 0, "pack")
        cross += int(vol[0].sum())
        LA.destroy()
        LB.destroy()
    assert cross == c1 <= c0
