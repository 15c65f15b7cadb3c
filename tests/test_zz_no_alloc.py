"""costa_volume_noalloc: the volume count for callers that cannot let the
library allocate device memory (their framework owns all device memory, or
they sit on a path where cudaMalloc's device synchronization is not
allowed).  It must give exactly the V of costa_volume, on repeated calls,
and reject pairs that do not fit its fixed scratch.

This file is collected last so that a failure here comes after every other
test has run; it also passes on its own in a fresh process."""
import numpy as np
import pytest

from workloads import configs as C
from workloads import layouts as L
from workloads.materialize import DeviceMatrix

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


def _pair(p, dev):
    import paper_2106_06601_gb300 as costa
    Bd = DeviceMatrix(p.B, p.dtype, dev)
    Ad = DeviceMatrix(p.A, p.dtype, dev)
    LA = costa.costa_layout_from_spec(p.A, p.dtype, Ad.block_ptrs())
    LB = costa.costa_layout_from_spec(p.B, p.dtype, Bd.block_ptrs())
    return (Ad, Bd), LA, LB


def test_noalloc_volume_matches_costa_volume():
    import paper_2106_06601_gb300 as costa
    dev = torch.device("cuda:0")
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream(dev).cuda_stream
    probs = [C.c1(), C.c2(), C.c5()] + [C.fuzz_problem(k) for k in range(40)]
    for p in probs:
        keep, LA, LB = _pair(p, dev)
        try:
            ref = costa.costa_volume(LA, LB, p.op, stream)
            first = costa.costa_volume_noalloc(LA, LB, p.op, stream)
            second = costa.costa_volume_noalloc(LA, LB, p.op, stream)
            assert np.array_equal(first, ref), p.name
            assert np.array_equal(second, ref), p.name
        finally:
            LA.destroy()
            LB.destroy()


def test_noalloc_rejects_pairs_beyond_its_scratch():
    import paper_2106_06601_gb300 as costa
    dev = torch.device("cuda:0")
    torch.cuda.set_device(dev)
    # P = 1024 ranks: V alone needs 8 MiB
    B = L.block_cyclic(1024, 1024, 1, 32, 1024, 1)
    A = L.block_cyclic(1024, 1024, 32, 1, 1, 1024)
    p = C.Problem("big-P", "f32", "N", 1.0, 0.0, A, B)
    keep, LA, LB = _pair(p, dev)
    try:
        with pytest.raises(costa.CostaError) as e:
            costa.costa_volume_noalloc(LA, LB, "N")
        assert e.value.status == 1 and "scratch" in str(e.value)
    finally:
        LA.destroy()
        LB.destroy()


def _scratch_need(P, nbrA, nbcA, nbr_op, nbc_op, nblkA, nblkB):
    """The scratch bytes a pair needs, by the rule stated in the header:
    8 P^2 for V, 8 bytes per split, 4 per block of A and of B, each section
    but the last rounded up to 256 bytes."""
    up = lambda x: (x + 255) // 256 * 256
    return (up(8 * P * P) + up(8 * (nbrA + 1)) + up(8 * (nbcA + 1)) + up(8 * (nbr_op + 1))
            + up(8 * (nbc_op + 1)) + up(4 * nblkA) + 4 * nblkB)


def _square_pair(P, k):
    """k x k blocks of size 1 on both sides (a k x k matrix), owners spread
    over P ranks with different patterns on the two sides."""
    idx = np.arange(k * k, dtype=np.int64)
    own_a = ((idx * 7 + 3) % P).astype(np.int32).reshape(k, k)
    own_b = ((idx * 5 + 1) % P).astype(np.int32).reshape(k, k)
    s = np.arange(k + 1, dtype=np.int64)
    A = L.packed_blocks(s, s, own_a, P)
    B = L.packed_blocks(s, s, own_b, P)
    return C.Problem("near-limit", "f32", "N", 1.0, 0.0, A, B)


def test_noalloc_allocates_nothing_and_limits_are_exact():
    """After a first call, repeated calls leave the device's free memory
    unchanged; a pair whose scratch need is just under 4 MiB matches
    costa_volume, and the next size up is rejected."""
    import paper_2106_06601_gb300 as costa
    dev = torch.device("cuda:0")
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream(dev).cuda_stream
    limit = 4 << 20
    P = 700
    k = 1
    while _scratch_need(P, k + 1, k + 1, k + 1, k + 1, (k + 1) ** 2, (k + 1) ** 2) <= limit:
        k += 1
    under = _square_pair(P, k)
    over = _square_pair(P, k + 1)
    assert _scratch_need(P, k, k, k, k, k * k, k * k) <= limit
    assert _scratch_need(P, k + 1, k + 1, k + 1, k + 1, (k + 1) ** 2, (k + 1) ** 2) > limit

    keep, LA, LB = _pair(under, dev)
    try:
        ref = costa.costa_volume(LA, LB, "N", stream)
        first = costa.costa_volume_noalloc(LA, LB, "N", stream)  # first call: set-up
        torch.cuda.synchronize(dev)
        free0, _ = torch.cuda.mem_get_info(dev)
        for _ in range(5):
            again = costa.costa_volume_noalloc(LA, LB, "N", stream)
            assert np.array_equal(again, ref)
        torch.cuda.synchronize(dev)
        free1, _ = torch.cuda.mem_get_info(dev)
        assert np.array_equal(first, ref)
        assert free1 == free0, (free0, free1)
    finally:
        LA.destroy()
        LB.destroy()

    keep, LA, LB = _pair(over, dev)
    try:
        with pytest.raises(costa.CostaError) as e:
            costa.costa_volume_noalloc(LA, LB, "N", stream)
        assert e.value.status == 1 and "scratch" in str(e.value)
    finally:
        LA.destroy()
        LB.destroy()
