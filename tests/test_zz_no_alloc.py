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
