"""TMA staging of the tile kernel's source tiles (COSTA_TMA=1, read when a
plan is built): in a fresh process with the variable set, the configurations
and fuzz problems take the TMA instance of the tile kernel and must give the
oracle's result (bit for bit in the exact class, else within the tolerance),
with no TMA wait giving up."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu
pytest.importorskip("torch")

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SCRIPT = r"""
import sys
import numpy as np
import torch
import oracle
import paper_2106_06601_gb300 as costa
from tests._gpu import OnDevice, compare
from workloads import configs as C
from workloads.materialize import DeviceMatrix
dev = torch.device("cuda:0")
torch.cuda.set_device(dev)
used = 0
for case in range(int(sys.argv[1])):
    p = C.fuzz_problem(case)
    g = OnDevice(p, dev, guard=2 if case % 3 == 0 else 0)
    g.run()
    compare(p, g.Ad.download(), g.oracle_result(), g.Ah, g.Bh)
    assert np.array_equal(g.Bd.download().arena, g.Bh.arena, equal_nan=True)
    st = costa.costa_debug_tma(g.LA, g.LB, p.op)
    assert st["timeouts"] == 0, st
    used += st["tiles"] + st["halves_tiles"]
    g.close()
for name in sys.argv[2:]:
    p = C.CONFIGS[name]() if name in C.CONFIGS else C.c2()
    if name == "c2beta":  # c2's layouts with a general beta: the kind TMA serves by default
        p.alpha, p.beta = -0.3, 0.7
    Bd = DeviceMatrix(p.B, p.dtype, dev).fill(p.b_kind, p.seed, p.src_stream)
    Ad = DeviceMatrix(p.A, p.dtype, dev).fill(p.a_kind, p.seed, p.tgt_stream)
    Bh, want = Bd.download(), Ad.download()
    Ad0 = want.copy()
    LA = costa.costa_layout_from_spec(p.A, p.dtype, Ad.block_ptrs())
    LB = costa.costa_layout_from_spec(p.B, p.dtype, Bd.block_ptrs())
    costa.costa_transform(LA, LB, p.op, p.alpha, p.beta, relabel=True,
                          stream=torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    st = costa.costa_debug_tma(LA, LB, p.op)
    assert st["timeouts"] == 0 and st["tiles"] + st["halves_tiles"] > 0, (name, st)
    oracle.transform(p.dtype, p.op, p.alpha, p.beta, p.A, want.buffers(), p.B, Bh.buffers())
    got = Ad.download()
    bad = 0
    for k in range(0, got.arena.size, 1 << 26):
        a, b = got.arena[k:k + (1 << 26)], want.arena[k:k + (1 << 26)]
        bad += int(a.size - np.count_nonzero((a == b) | (np.isnan(a) & np.isnan(b))))
    if name == "c2beta":
        from tests._util import assert_close, global_matrix, op_apply
        al, be = oracle.scalar(p.dtype, p.alpha), oracle.scalar(p.dtype, p.beta)
        X = op_apply(p.op, global_matrix(p.B, Bh.buffers()))
        A0 = global_matrix(p.A, Ad0.buffers())
        assert_close(p.dtype, global_matrix(p.A, got.buffers()), global_matrix(p.A, want.buffers()),
                     al, be, X, A0, exact=False)
    else:
        assert bad == 0, (name, bad)
    LA.destroy(); LB.destroy()
    print(name, st, flush=True)
print("tma tiles used in fuzz cases:", used)
"""


def test_tma_staging_matches_oracle():
    """COSTA_TMA=1: every kind and type through the TMA instance."""
    env = dict(os.environ, COSTA_TMA="1")
    r = subprocess.run([sys.executable, "-c", SCRIPT, "60", "c2", "c3", "c5"], cwd=ROOT, env=env,
                       capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, (r.stdout[-3000:], r.stderr[-3000:])
    assert "tma tiles used" in r.stdout


def test_default_policy_picks_the_measured_cases():
    """Without COSTA_TMA: the f64 plans (c2, c5) hold TMA tiles in their
    direct list for the general axpby kind only, none in the x-halves list;
    c3 (c128) holds none."""
    script = r"""
import torch
import paper_2106_06601_gb300 as costa
from workloads import configs as C
from workloads.materialize import DeviceMatrix
dev = torch.device("cuda:0")
for name in ("c2", "c5", "c3"):
    p = C.CONFIGS[name]()
    Bd = DeviceMatrix(p.B, p.dtype, dev)
    Ad = DeviceMatrix(p.A, p.dtype, dev)
    LA = costa.costa_layout_from_spec(p.A, p.dtype, Ad.block_ptrs())
    LB = costa.costa_layout_from_spec(p.B, p.dtype, Bd.block_ptrs())
    st = costa.costa_debug_tma(LA, LB, p.op)
    print(name, st["tiles"], st["halves_tiles"], st["kinds"], st["halves_kinds"], st["timeouts"])
    LA.destroy(); LB.destroy(); del Ad, Bd; costa.costa_release_plans(); torch.cuda.empty_cache()
"""
    env = dict(os.environ)
    env.pop("COSTA_TMA", None)
    r = subprocess.run([sys.executable, "-c", script], cwd=ROOT, env=env, capture_output=True,
                       text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-3000:]
    rows = {line.split()[0]: [int(x) for x in line.split()[1:]] for line in r.stdout.splitlines()}
    K_AXPBY = 2
    for name in ("c2", "c5"):
        assert rows[name][0] > 0 and rows[name][1] == 0, rows
        assert rows[name][2] == 1 << K_AXPBY and rows[name][3] == 0, rows
    assert rows["c3"][:4] == [0, 0, 0, 0]
    assert all(v[4] == 0 for v in rows.values())


def test_default_policy_general_beta_matches_oracle():
    """The default policy's own case: f64 with a general beta (c2's layouts,
    beta = 0.7) through the TMA instance, against the oracle within the
    tolerance."""
    env = dict(os.environ)
    env.pop("COSTA_TMA", None)
    r = subprocess.run([sys.executable, "-c", SCRIPT, "0", "c2beta"], cwd=ROOT, env=env,
                       capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, (r.stdout[-3000:], r.stderr[-3000:])
    assert "c2beta" in r.stdout


def test_lists_built_after_capture_keep_the_graph_valid():
    """The TMA-staged lists are built by the first eager call of a kind that
    uses them, never inside a stream capture.  A general-beta f64 transform
    captured in a CUDA graph before that call replays on the cp.async lists;
    the eager call then builds the TMA lists (and takes them), and the graph
    still replays correctly afterwards.  Every step is compared with the
    oracle applied to the A it started from, within the tolerance."""
    script = r"""
import numpy as np
import torch
import oracle
import paper_2106_06601_gb300 as costa
from tests._util import assert_close, global_matrix, op_apply
from workloads import configs as C
from workloads.materialize import DeviceMatrix
dev = torch.device("cuda:0")
torch.cuda.set_device(dev)
p = C.c2(2048)
p.alpha, p.beta = -0.3, 0.7
Bd = DeviceMatrix(p.B, p.dtype, dev).fill(p.b_kind, p.seed, p.src_stream)
Ad = DeviceMatrix(p.A, p.dtype, dev).fill(p.a_kind, p.seed, p.tgt_stream)
Bh = Bd.download()
LA = costa.costa_layout_from_spec(p.A, p.dtype, Ad.block_ptrs())
LB = costa.costa_layout_from_spec(p.B, p.dtype, Bd.block_ptrs())
al, be = oracle.scalar(p.dtype, p.alpha), oracle.scalar(p.dtype, p.beta)
X = op_apply(p.op, global_matrix(p.B, Bh.buffers()))
s = torch.cuda.Stream(dev)
costa.costa_plan_stats_get(LA, LB, p.op, relabel=True)  # the plan, without a transform
graph = torch.cuda.CUDAGraph()
with torch.cuda.graph(graph, stream=s):
    costa.costa_transform(LA, LB, p.op, p.alpha, p.beta, relabel=True,
                          stream=torch.cuda.current_stream().cuda_stream)

def step(run):
    before = Ad.download()
    run()
    torch.cuda.synchronize(dev)
    want = before.copy()
    oracle.transform(p.dtype, p.op, p.alpha, p.beta, p.A, want.buffers(), p.B, Bh.buffers())
    got = Ad.download()
    assert_close(p.dtype, global_matrix(p.A, got.buffers()), global_matrix(p.A, want.buffers()),
                 al, be, X, global_matrix(p.A, before.buffers()), exact=False)

step(graph.replay)
step(graph.replay)
step(lambda: costa.costa_transform(LA, LB, p.op, p.alpha, p.beta, relabel=True, stream=s.cuda_stream))
st = costa.costa_debug_tma(LA, LB, p.op)
assert st["tiles"] > 0 and st["timeouts"] == 0, st
step(graph.replay)
step(lambda: costa.costa_transform(LA, LB, p.op, p.alpha, p.beta, relabel=True, stream=s.cuda_stream))
print("ok", st)
"""
    env = dict(os.environ)
    env.pop("COSTA_TMA", None)
    r = subprocess.run([sys.executable, "-c", script], cwd=ROOT, env=env, capture_output=True,
                       text=True, timeout=600)
    assert r.returncode == 0, (r.stdout[-3000:], r.stderr[-3000:])
    assert "ok" in r.stdout
