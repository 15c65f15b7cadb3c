"""COSTA_LOG: with COSTA_LOG=2 a process logs its plans, relabelings and
transform calls on stderr (lines prefixed "[costa] "); without it, nothing."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu
pytest.importorskip("torch")

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SCRIPT = """
import torch
import paper_2106_06601_gb300 as costa
from tests._gpu import OnDevice
from workloads import configs as C
dev = torch.device("cuda:0")
g = OnDevice(C.c1(), dev)
g.run(relabel=True)
g.run(relabel=True, mode="message")
g.close()
"""


def _run(level):
    env = dict(os.environ)
    env.pop("COSTA_LOG", None)
    if level is not None:
        env["COSTA_LOG"] = str(level)
    r = subprocess.run([sys.executable, "-c", SCRIPT], cwd=ROOT, env=env, capture_output=True,
                       text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    return [line for line in r.stderr.splitlines() if line.startswith("[costa] ")]


def test_costa_log_levels():
    lines = _run(2)
    text = "\n".join(lines)
    for what in ("plan:", "relabel:", "message plan", "transform:"):
        assert f"[costa] {what}" in text, text
    assert sum("transform:" in line for line in lines) == 2
    one = _run(1)
    assert one and not any("transform:" in line for line in one)
    assert _run(None) == []
