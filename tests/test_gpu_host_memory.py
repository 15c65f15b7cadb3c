"""Storage in host memory.  Blocks may live in host memory allocated or
registered with CUDA (pinned); the kernels then read and write it directly
over the host link, and the results equal the oracle's exactly as for device
storage.  Pageable host memory is rejected when the plan is built, before any
kernel touches a block (the check runs through costa_plan_stats_get, whose
only kernel, the volume count, reads layout tables and no block)."""
import numpy as np
import pytest

import paper_2106_06601_gb300 as costa
from tests._gpu import compare
from workloads import configs as C
from workloads.materialize import HostMatrix, block_element_offsets

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def dev():
    d = torch.device("cuda:0")
    torch.cuda.set_device(d)
    return d


def _pinned(host: HostMatrix):
    t = torch.from_numpy(host.arena).pin_memory()
    assert t.is_pinned()
    return t


def _ptrs(spec, host: HostMatrix, arena_tensor):
    off = block_element_offsets(spec, host.starts)
    return (arena_tensor.data_ptr() + off * arena_tensor.element_size()).astype(np.uint64)


@pytest.mark.parametrize("case", [3, 9, 21, 40, 55, 77])
@pytest.mark.parametrize("mode", ["direct", "message"])
def test_pinned_host_storage_matches_oracle(case, mode, dev):
    p = C.fuzz_problem(case)
    Bh = HostMatrix(p.B, p.dtype).fill(p.b_kind, p.seed, p.src_stream)
    Ah = HostMatrix(p.A, p.dtype).fill(p.a_kind, p.seed, p.tgt_stream)
    Bt, At = _pinned(Bh), _pinned(Ah)
    LA = costa.costa_layout_from_spec(p.A, p.dtype, _ptrs(p.A, Ah, At))
    LB = costa.costa_layout_from_spec(p.B, p.dtype, _ptrs(p.B, Bh, Bt))
    try:
        stream = torch.cuda.current_stream(dev).cuda_stream
        costa.costa_transform(LA, LB, p.op, p.alpha, p.beta, relabel=True, stream=stream, mode=mode)
        torch.cuda.synchronize(dev)
        got = HostMatrix.__new__(HostMatrix)
        got.spec, got.dtype, got.guard, got.starts = p.A, p.dtype, 0, Ah.starts
        got.arena = At.numpy().copy()
        want = Ah.copy()
        import oracle
        oracle.transform(p.dtype, p.op, p.alpha, p.beta, p.A, want.buffers(), p.B, Bh.buffers())
        compare(p, got, want, Ah, Bh)
        assert np.array_equal(Bt.numpy(), Bh.arena, equal_nan=True)  # B is read-only
    finally:
        LA.destroy()
        LB.destroy()


def test_pageable_host_storage_is_rejected(dev):
    from workloads.materialize import DeviceMatrix
    p = C.fuzz_problem(3)
    Bh = HostMatrix(p.B, p.dtype).fill(p.b_kind, p.seed, p.src_stream)
    Ad = DeviceMatrix(p.A, p.dtype, dev)
    LA = costa.costa_layout_from_spec(p.A, p.dtype, Ad.block_ptrs())
    # B's blocks point into a plain numpy array: pageable memory
    LB = costa.costa_layout_from_spec(p.B, p.dtype, _ptrs(p.B, Bh, torch.from_numpy(Bh.arena)))
    try:
        with pytest.raises(costa.CostaError) as e:
            costa.costa_plan_stats_get(LA, LB, p.op, relabel=True,
                                       stream=torch.cuda.current_stream(dev).cuda_stream)
        assert e.value.status == 2 and "pageable" in str(e.value)
    finally:
        LA.destroy()
        LB.destroy()
