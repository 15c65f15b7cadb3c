"""Calls on one layout pair from two streams.

A plan's device scratch (the per-problem scalars of a batch whose scalars
differ, and message mode's staging buffer) is shared by every call on the
plan.  The library orders the calls that use it in call order: a call on
another stream than the previous such call waits for that call's completion
event.  Here call 1 is held back on stream 1 behind a long sleep kernel while
call 2, with other scalars, is issued on stream 2 with no ordering from the
caller.  Both are in the bit-exact class (power-of-two scalars), so the
result must be the oracle's call 2 applied after call 1, bit for bit.
"""
import numpy as np
import pytest

import oracle
from tests._gpu import OnDevice
from workloads import configs as C

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")

SLEEP_CYCLES = 200_000_000  # about 0.1 s at 2 GHz


@pytest.fixture(scope="module")
def dev():
    d = torch.device("cuda:0")
    torch.cuda.set_device(d)
    return d


def _problems(n):
    probs = []
    for k in range(n):
        p = C.fuzz_problem(500 + k, dtype="f64", P=4)
        p.a_kind = "uniform"
        probs.append(p)
    return probs


def _run_two_streams(dev, gs, probs, first, second, mode):
    import paper_2106_06601_gb300 as costa
    As, Bs, ops = [g.LA for g in gs], [g.LB for g in gs], [p.op for p in probs]
    costa.costa_plan_stats_get(As, Bs, ops, relabel=True)  # plan built before the race
    if mode == "message":
        # the staging buffer is allocated by the first message-mode call
        costa.costa_transform_batched(As, Bs, ops, [1.0] * len(gs), [0.0] * len(gs), relabel=True,
                                      stream=torch.cuda.current_stream().cuda_stream, mode=mode)
        torch.cuda.synchronize(dev)
        for g in gs:
            g.reset_A()
        torch.cuda.synchronize(dev)
    s1, s2 = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    with torch.cuda.stream(s1):
        torch.cuda._sleep(SLEEP_CYCLES)
    costa.costa_transform_batched(As, Bs, ops, first[0], first[1], relabel=True,
                                  stream=s1.cuda_stream, mode=mode)
    costa.costa_transform_batched(As, Bs, ops, second[0], second[1], relabel=True,
                                  stream=s2.cuda_stream, mode=mode)
    torch.cuda.synchronize(dev)


def _check(gs, probs, first, second):
    for k, (g, p) in enumerate(zip(gs, probs)):
        want = g.Ah.copy()
        for al, be in ((first[0][k], first[1][k]), (second[0][k], second[1][k])):
            oracle.transform(p.dtype, p.op, al, be, p.A, want.buffers(), p.B, g.Bh.buffers())
        got = g.Ad.download()
        assert np.array_equal(got.arena, want.arena, equal_nan=True), f"problem {k}"


def test_batched_scalars_two_streams(dev):
    """Per-problem scalars differ within each batch and between the calls."""
    probs = _problems(6)
    gs = [OnDevice(p, dev) for p in probs]
    try:
        first = ([2.0 ** (k % 3) for k in range(6)], [0.5 if k % 2 else 2.0 for k in range(6)])
        second = ([0.5 * (-1) ** k for k in range(6)], [-2.0 ** -(k % 3) for k in range(6)])
        _run_two_streams(dev, gs, probs, first, second, "direct")
        _check(gs, probs, first, second)
    finally:
        for g in gs:
            g.close()


def test_message_mode_two_streams(dev):
    """Message mode's pack, local and unpack phases share the staging
    buffer; uniform scalars, different between the calls."""
    probs = _problems(3)
    gs = [OnDevice(p, dev) for p in probs]
    try:
        first = ([2.0] * 3, [0.5] * 3)
        second = ([-0.5] * 3, [4.0] * 3)
        _run_two_streams(dev, gs, probs, first, second, "message")
        _check(gs, probs, first, second)
    finally:
        for g in gs:
            g.close()
