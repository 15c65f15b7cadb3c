"""The multi-GPU exchange's kernels on one GB300 (Sec. 6 "Implementation",
Alg. 3): G processes are emulated on the one device, each with its own
layouts (NULL pointers for the blocks of ranks on other processes), its own
exchange and its own send and receive buffers.  Every process packs, the
segments are copied to their receivers on the device (the all-to-all-v a
multi-GPU run does with NCCL), and every process runs its local and unpack
lists.  No kernel waits on another process's kernels.  A must equal the
oracle's result bit for bit (beta = 0 or power-of-two scalars) or within the
tolerance of tests/_util (other scalars), and nothing outside A's blocks may
change."""
import numpy as np
import pytest

import oracle
from tests._exchange import block_placement
from tests._gpu import OnDevice, compare
from workloads import configs as C
from workloads.materialize import DeviceMatrix, block_element_offsets

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def dev():
    d = torch.device("cuda:0")
    torch.cuda.set_device(d)
    return d


def _ptrs(spec, dm: DeviceMatrix, place, g):
    off = block_element_offsets(spec, dm.starts)
    ptr = (dm.arena.data_ptr() + off * dm.esize).astype(np.uint64)
    return np.where(np.asarray(place)[spec.owner] == g, ptr, np.uint64(0))


def run_exchange(p, Ad, Bd, G, place, dev):
    """All G processes' phases on one device; returns the kernel launches."""
    import paper_2106_06601_gb300 as costa
    stream = torch.cuda.current_stream(dev).cuda_stream
    procs = []
    for g in range(G):
        LA = costa.costa_layout_from_spec(p.A, p.dtype, _ptrs(p.A, Ad, place, g))
        LB = costa.costa_layout_from_spec(p.B, p.dtype, _ptrs(p.B, Bd, place, g))
        sb, rb = costa.costa_exchange_sizes(LA, LB, p.op, G, place, g)
        send = torch.empty(max(16, int(sb.sum())), dtype=torch.uint8, device=dev)
        recv = torch.empty(max(16, int(rb.sum())), dtype=torch.uint8, device=dev)
        x = costa.Exchange(LA, LB, p.op, G, place, g, send.data_ptr(), recv.data_ptr())
        assert all(np.array_equal(a, b) for a, b in zip(x.counts(), (sb, rb)))
        procs.append((LA, LB, sb, rb, send, recv, x))
    n0 = costa.costa_kernel_launch_count()
    for (_, _, _, _, _, _, x) in procs:
        x.pack(stream)
    for g in range(G):
        rb, recv = procs[g][3], procs[g][5]
        rd = np.concatenate([[0], np.cumsum(rb)[:-1]])
        for h in range(G):
            sb, send = procs[h][2], procs[h][4]
            sd = np.concatenate([[0], np.cumsum(sb)[:-1]])
            n = int(rb[h])
            assert n == int(sb[g])
            if n:
                recv[rd[h]:rd[h] + n].copy_(send[sd[g]:sd[g] + n])
    for (_, _, _, _, _, _, x) in procs:
        x.local(p.alpha, p.beta, stream)
        x.unpack(p.alpha, p.beta, stream)
    torch.cuda.synchronize(dev)
    launches = costa.costa_kernel_launch_count() - n0
    for (LA, LB, _, _, _, _, x) in procs:
        x.destroy()
        LA.destroy()
        LB.destroy()
    return launches


def check(p, G, place, dev, guard=0):
    g = OnDevice(p, dev, guard=guard)
    try:
        launches = run_exchange(p, g.Ad, g.Bd, G, place, dev)
        assert launches > 0
        compare(p, g.Ad.download(), g.oracle_result(), g.Ah, g.Bh)
        assert np.array_equal(g.Bd.download().arena, g.Bh.arena, equal_nan=True)
    finally:
        g.close()


SCALARS = [(1.0, 0.0), (2.0, 0.5), (-0.5, 0.0), (0.5, -2.0)]


@pytest.mark.parametrize("case", range(40))
def test_exchange_fuzz(case, dev):
    p = C.fuzz_problem(600 + case)
    p.alpha, p.beta = SCALARS[case % len(SCALARS)]
    p.a_kind = "nan" if p.beta == 0 else "uniform"
    P = p.A.nranks
    G = (2, 3, 4, 1)[case % 4]
    if case % 3 == 0:
        place = block_placement(P, G)
    else:
        place = np.random.default_rng(case).integers(0, G, P).astype(np.int32)
    check(p, G, place, dev, guard=3 if case % 5 == 0 else 0)


@pytest.mark.parametrize("case", range(12))
def test_exchange_small_blocks(case, dev):
    """Small and odd blocks: the lists take the small-tile kernel and the
    misaligned instance."""
    p = C.small_block_problem(case * 7)
    check(p, 2 + case % 3, block_placement(p.A.nranks, 2 + case % 3), dev)


@pytest.mark.parametrize("name,G", [("c2", 4), ("c3", 8), ("c5", 8)])
def test_exchange_configs_full_size(name, G, dev):
    """The configurations at full size with their ranks in G blocks (inputs
    filled on the device), every element compared with the oracle."""
    p = C.CONFIGS[name]()
    Bd = DeviceMatrix(p.B, p.dtype, dev).fill(p.b_kind, p.seed, p.src_stream)
    Ad = DeviceMatrix(p.A, p.dtype, dev).fill(p.a_kind, p.seed, p.tgt_stream)
    Bh, want = Bd.download(), Ad.download()
    run_exchange(p, Ad, Bd, G, block_placement(p.A.nranks, G), dev)
    oracle.transform(p.dtype, p.op, p.alpha, p.beta, p.A, want.buffers(), p.B, Bh.buffers())
    got = Ad.download()
    bad = 0
    for k in range(0, got.arena.size, 1 << 26):
        g, w = got.arena[k:k + (1 << 26)], want.arena[k:k + (1 << 26)]
        bad += int(g.size - np.count_nonzero((g == w) | (np.isnan(g) & np.isnan(w))))
    assert bad == 0, f"{name}: {bad} elements differ"
    assert np.array_equal(Bd.download().arena, Bh.arena)
