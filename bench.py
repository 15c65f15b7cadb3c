"""Benchmark of the reshuffle A = alpha * op(B) + beta * A on GB300.

Headline workload: c5, the largest single-GPU configuration (12.9 GB moved per
call): B 131072 x 4096 f64 normal(0, 1), block-cyclic 32x32 on a 16x16 grid ->
A 4096 x 131072 in 256 row panels of 16 rows (a COSMA-style blocked layout,
one panel per rank), op = T, alpha = beta = 1, P = 256 virtual ranks,
relabeling on.  The same line carries c2, c3 and c4 under `per_config`, each
with the headline's fields.  One step = one costa_transform (or
costa_transform_batched) call in direct mode through the C ABI; its plan
(overlay, volume kernel, relabeling, tile lists) is built once before the
timed region and reported separately, like a reused transformer.

Prints one JSON line.  `value` = algorithmic bytes (read B + read A if
beta != 0 + write A) of all ranks / max-over-ranks device time.  `e2e` = the
same metric through the same call with the matrices in pinned host memory
(the kernels read and write them over the host link), and under `copies`
with explicit host->device and device->host copies around the call.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload c5|c2|c3|c4|c1|...]
                  [--also c2,c3,c4|none] [--mode direct|message] [--impl gb300|reference]

Multi-GPU (torchrun, N > 1): a single-problem workload is split over the N
GPUs (the multi-GPU exchange: ranks in blocks of P / N per GPU, A's owners
relabeled for that placement, pack -> NCCL all-to-all-v -> unpack), total work
fixed ("strong"); the batched c4 runs one independent replica per GPU
("weak").  --exchange runs the exchange path on one GPU too.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import platform
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from workloads import configs as C  # noqa: E402
from workloads.materialize import DeviceMatrix, HostMatrix  # noqa: E402

L2_BYTES = 129 * 1024 * 1024
KERNEL_SOURCES = ["paper_2106_06601_gb300/csrc/remap_impl.cuh",
                  "paper_2106_06601_gb300/csrc/fxdot.h",  # fixed-point sums of the complex kinds
                  "paper_2106_06601_gb300/csrc/remap_f64.cu",
                  "paper_2106_06601_gb300/csrc/remap_f32.cu",
                  "paper_2106_06601_gb300/csrc/remap_c64.cu",
                  "paper_2106_06601_gb300/csrc/remap_c128.cu",
                  "paper_2106_06601_gb300/csrc/tiles.cpp",  # tile lists, their order, small-tile pieces
                  "paper_2106_06601_gb300/csrc/tiles.h"]


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=500)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--workload", default="c5", choices=list(C.CONFIGS) + list(C.EXTRA_WORKLOADS))
    ap.add_argument("--also", default="auto",
                    help="comma-separated workloads measured after the headline and reported "
                         "under per_config ('auto': c2,c3,c4 when the headline is c5; 'none')")
    ap.add_argument("--mode", default="direct", choices=["direct", "message"])
    ap.add_argument("--exchange", action="store_true",
                    help="run the multi-GPU exchange path also on one GPU (it is the path "
                         "for every single-problem workload when N > 1)")
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--e2e-steps", type=int, default=20)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--small", action="store_true",
                    help="same layouts at about 1 GB (for profiler captures only)")
    return ap.parse_args()


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def code_only(text: str) -> str:
    """C/C++ source without its comments and blank lines (string literals
    are kept whole), so that editing a comment keeps recorded profiles."""
    out, i, n = [], 0, len(text)
    while i < n:
        c = text[i]
        if c == '"':
            j = i + 1
            while j < n and text[j] != '"':
                j += 2 if text[j] == "\\" else 1
            out.append(text[i:j + 1])
            i = j + 1
        elif text.startswith("//", i):
            while i < n and text[i] != "\n":
                i += 1
        elif text.startswith("/*", i):
            j = text.find("*/", i + 2)
            i = n if j < 0 else j + 2
        else:
            out.append(c)
            i += 1
    lines = (line.rstrip() for line in "".join(out).split("\n"))
    return "\n".join(line for line in lines if line)


def kernel_hash() -> str:
    """Hash of the code (comments aside) of the remap kernels and of the tile
    lists they walk."""
    h = hashlib.sha256()
    for f in KERNEL_SOURCES:
        with open(os.path.join(ROOT, f), encoding="utf-8") as fh:
            h.update(code_only(fh.read()).encode())
    return h.hexdigest()[:16]


def recorded_traffic(workload: str):
    """DRAM bytes per launch from the committed ncu summary of this workload,
    if it was taken on the current kernel sources."""
    path = os.path.join(ROOT, "profiles", f"remap_{workload}_traffic.json")
    try:
        with open(path) as f:
            d = json.load(f)
        if d.get("kernel_sources_sha256_16") == kernel_hash():
            return d.get("dram_bytes_per_launch")
    except Exception:
        pass
    return None


class ClockSampler:
    """nvidia-smi clocks and throttle reasons, sampled every 100 ms."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.samples = []
        self.proc = None
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(gpu_index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.samples.append((time.time(), [x.strip() for x in line.split(",")]))

    def stop(self):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self, t0, t1):
        if not self.proc:
            return None
        win = [s for t, s in self.samples if t0 <= t <= t1]
        window = "timed"
        if not win:
            win = [s for _, s in self.samples]
            window = "whole run"
        if not win:
            return None
        sm = []
        reasons = set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        smax = None
        for s in win:
            try:
                sm.append(float(s[1]))
                smax = float(s[2])
            except ValueError:
                continue
            for k, nm in enumerate(names):
                if len(s) > 5 + k and s[5 + k].lower().startswith("active"):
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": smax,
                "reasons": sorted(reasons), "samples": len(sm), "window": window}


def max_over_ranks(x: float, device=None) -> float:
    """The maximum of x over all ranks (identity without a process group)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(bytes_per_rank: int, world: int, steps: int, max_ms: float) -> float:
    """Whole-job GB/s: the bytes every rank moved in `steps` steps over the
    slowest rank's time."""
    return bytes_per_rank * world * steps / (max_ms * 1e-3) / 1e9


def problems(workload, small=False):
    p = (C.CONFIGS_SMALL if small else {**C.CONFIGS, **C.EXTRA_WORKLOADS})[workload]()
    return p if isinstance(p, list) else [p]


def esize(dtype):
    return {"f32": 4, "f64": 8, "c64": 8, "c128": 16}[dtype]


def algorithmic_bytes(probs) -> int:
    return sum(p.algorithmic_bytes() for p in probs)


def run_gpu(args, workload, rank, world, local_rank):
    import torch
    import paper_2106_06601_gb300 as costa

    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    probs = problems(workload, args.small)
    mats = []
    for p in probs:
        Bd = DeviceMatrix(p.B, p.dtype, dev).fill(p.b_kind, p.seed, p.src_stream)
        Ad = DeviceMatrix(p.A, p.dtype, dev).fill(p.a_kind, p.seed, p.tgt_stream)
        LA = costa.costa_layout_from_spec(p.A, p.dtype, Ad.block_ptrs())
        LB = costa.costa_layout_from_spec(p.B, p.dtype, Bd.block_ptrs())
        mats.append((p, Bd, Ad, LA, LB))
    stream = torch.cuda.Stream(dev)
    sh = stream.cuda_stream
    As = [m[3] for m in mats]
    Bs = [m[4] for m in mats]
    ops = [p.op for p in probs]
    alphas = [p.alpha for p in probs]
    betas = [p.beta for p in probs]
    batched = len(probs) > 1

    def step():
        if batched:
            costa.costa_transform_batched(As, Bs, ops, alphas, betas, relabel=True, stream=sh,
                                          mode=args.mode)
        else:
            costa.costa_transform(As[0], Bs[0], ops[0], alphas[0], betas[0], relabel=True,
                                  stream=sh, mode=args.mode)

    # plan (overlay, volume kernel, relabeling, tiles): built once, timed apart
    t0 = time.perf_counter()
    stats = costa.costa_plan_stats_get(As, Bs, ops, relabel=True, stream=sh)
    plan_s = time.perf_counter() - t0
    with torch.cuda.stream(stream):
        for _ in range(max(3, args.warmup)):
            step()
    torch.cuda.synchronize(dev)
    if args.mode == "message":
        stats = costa.costa_plan_stats_get(As, Bs, ops, relabel=True, stream=sh)

    nbytes = algorithmic_bytes(probs)
    clocks = ClockSampler(local_rank)
    time.sleep(0.3)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize(dev)
    n0 = costa.costa_kernel_launch_count()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t_wall0 = time.time()
    with torch.cuda.stream(stream):
        start.record(stream)
        for k in range(args.steps):
            ev[k][0].record(stream)
            step()
            ev[k][1].record(stream)
        end.record(stream)
    torch.cuda.synchronize(dev)
    t_wall1 = time.time()
    if world > 1:
        torch.distributed.barrier()
    launches = costa.costa_kernel_launch_count() - n0
    total_ms = start.elapsed_time(end)
    per = [a.elapsed_time(b) for a, b in ev]
    clocks.stop()
    clk = clocks.summary(t_wall0, t_wall1)

    total_ms = max_over_ranks(total_ms, dev)
    ms_per_step = total_ms / args.steps
    value = job_throughput(nbytes, world, args.steps, total_ms)

    # ---- end to end: storage in pinned host memory ----
    e2e = None
    if args.e2e_steps > 0:
        e2e = run_e2e(args, costa, mats, step, stream, dev, world, nbytes)

    phases = None
    if args.mode == "message":
        phases = message_phases(args, probs, stats, step, stream, dev)
    kernels = direct_kernels(costa, mats)
    for m in mats:
        m[3].destroy()
        m[4].destroy()
    peak, peak_kind = measured_peaks()
    avg_launch_ms = statistics.mean(per)
    achieved = nbytes / (avg_launch_ms * 1e-3) / 1e9
    traffic = recorded_traffic(workload) if args.mode == "direct" else None
    return dict(value=value, ms_per_step=ms_per_step, total_ms=total_ms, per=per,
                launches=launches, clocks=clk, e2e=e2e, plan_s=plan_s, stats=stats,
                nbytes=nbytes, achieved=achieved, peak=peak, peak_kind=peak_kind,
                traffic=traffic, probs=probs, phases=phases, kernels=kernels)


def run_exchange(args, workload, rank, world, local_rank):
    """The reshuffle split over the job's GPUs (Sec. 6 "Implementation", Alg.
    3): the P ranks in blocks of about P / N per GPU, A's owners relabeled for
    that placement (costa_relabel_placement), and every step = pack, local
    remap, an NCCL all-to-all-v of the packed segments, unpack.  value = the
    algorithmic bytes of the whole matrix (all GPUs) / the slowest rank's
    time: total work fixed as N grows ("strong")."""
    import dataclasses
    import torch
    import torch.distributed as dist
    import paper_2106_06601_gb300 as costa
    from workloads.materialize import block_element_offsets

    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    probs = problems(workload, args.small)
    assert len(probs) == 1
    p = probs[0]
    P, G, g = p.A.nranks, world, rank
    place = np.array([r * G // P for r in range(P)], dtype=np.int32)
    t0 = time.perf_counter()
    Bd = DeviceMatrix(p.B, p.dtype, dev).fill(p.b_kind, p.seed, p.src_stream)

    def ptrs(spec, dm):  # NULL for the blocks of ranks on other GPUs
        off = block_element_offsets(spec, dm.starts)
        ptr = (dm.arena.data_ptr() + off * dm.esize).astype(np.uint64)
        return np.where(place[spec.owner] == g, ptr, np.uint64(0))

    # relabeling for the placement: label q's blocks go to process sigma(q)
    LA0 = costa.costa_layout_from_spec(p.A, p.dtype, np.zeros(p.A.owner.size, np.uint64))
    LB = costa.costa_layout_from_spec(p.B, p.dtype, ptrs(p.B, Bd))
    tv = time.perf_counter()
    V = costa.costa_volume_noalloc(LA0, LB, p.op, 0)
    volume_ms = (time.perf_counter() - tv) * 1e3
    tr = time.perf_counter()
    sigma, cross0, cross1 = costa.costa_relabel_placement(V, G, place, 0.0)
    relabel_ms = (time.perf_counter() - tr) * 1e3
    LA0.destroy()
    A = dataclasses.replace(p.A, owner=sigma[p.A.owner].astype(np.int32))
    Ad = DeviceMatrix(A, p.dtype, dev).fill(p.a_kind, p.seed, p.tgt_stream)
    LA = costa.costa_layout_from_spec(A, p.dtype, ptrs(A, Ad))
    sb, rb = costa.costa_exchange_sizes(LA, LB, p.op, G, place, g)
    if world > 1:  # sends and receives must pair up before any NCCL call
        allc = [torch.zeros(2 * G, dtype=torch.int64, device=dev) for _ in range(G)]
        dist.all_gather(allc, torch.from_numpy(np.concatenate([sb, rb])).to(dev))
        allc = torch.stack(allc).cpu().numpy()
        if not all(allc[a, b] == allc[b, G + a] for a in range(G) for b in range(G)):
            raise RuntimeError("exchange segment sizes do not pair up across ranks")
    send = torch.empty(max(16, int(sb.sum())), dtype=torch.uint8, device=dev)
    recv = torch.empty(max(16, int(rb.sum())), dtype=torch.uint8, device=dev)
    x = costa.Exchange(LA, LB, p.op, G, place, g, send.data_ptr(), recv.data_ptr())
    plan_s = time.perf_counter() - t0
    stream = torch.cuda.Stream(dev)
    sh = stream.cuda_stream
    sbl, rbl = sb.tolist(), rb.tolist()

    def step(ev=None):
        if ev is not None:
            ev[0].record(stream)
        x.pack(sh)
        x.local(p.alpha, p.beta, sh)
        if ev is not None:
            ev[1].record(stream)
        if world > 1:
            dist.all_to_all_single(recv, send, rbl, sbl)
        if ev is not None:
            ev[2].record(stream)
        x.unpack(p.alpha, p.beta, sh)
        if ev is not None:
            ev[3].record(stream)

    with torch.cuda.stream(stream):
        for _ in range(max(3, args.warmup)):
            step()
    torch.cuda.synchronize(dev)
    clocks = ClockSampler(local_rank)
    time.sleep(0.3)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    n0 = costa.costa_kernel_launch_count()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t_wall0 = time.time()
    with torch.cuda.stream(stream):
        start.record(stream)
        for k in range(args.steps):
            ev[k][0].record(stream)
            step()
            ev[k][1].record(stream)
        end.record(stream)
    torch.cuda.synchronize(dev)
    t_wall1 = time.time()
    if world > 1:
        dist.barrier()
    launches = costa.costa_kernel_launch_count() - n0
    total_ms = max_over_ranks(start.elapsed_time(end), dev)
    per = [a.elapsed_time(b) for a, b in ev]
    clocks.stop()
    clk = clocks.summary(t_wall0, t_wall1)
    nbytes = p.algorithmic_bytes()
    # phases (after the timed region): pack + local, the exchange, unpack
    n = max(10, min(args.steps, 100))
    pev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(n)]
    with torch.cuda.stream(stream):
        for k in range(n):
            step(pev[k])
    torch.cuda.synchronize(dev)
    es = p.esize
    ra = 1 if p.beta != 0 else 0
    phase = {}
    for name, a, b in (("pack+local", 0, 1), ("exchange", 1, 2), ("unpack", 2, 3)):
        phase[name] = statistics.mean(e[a].elapsed_time(e[b]) for e in pev)
    send_b, recv_b = int(sb.sum()), int(rb.sum())
    # elements of this GPU's tiles, from V and the relabeling: source rank p
    # on GPU place[p], target label q on GPU place[sigma[q]]
    src_here = place == g
    tgt_here = place[sigma] == g
    local_el = int(V[np.ix_(src_here, tgt_here)].sum())
    sent_el = int(V[np.ix_(src_here, ~tgt_here)].sum())
    recv_el = int(V[np.ix_(~src_here, tgt_here)].sum())
    # algorithmic bytes of this GPU's kernels: pack reads and writes each sent
    # element; local and unpack read the source, A when beta != 0, write A
    kernel_bytes = es * (2 * sent_el + (2 + ra) * (local_el + recv_el))
    e2e = run_exchange_e2e(args, step, stream, dev, world, nbytes, Bd, Ad, p, A, place, g)
    x.destroy()
    LA.destroy()
    LB.destroy()
    peak, peak_kind = measured_peaks()
    value = job_throughput(nbytes, 1, args.steps, total_ms)
    stats = {"total_volume": p.A.m * p.A.n, "local_identity": int(np.trace(V)),
             "local_relabeled": int(sum(int(V[sigma[q], q]) for q in range(P))),
             "n_cells": None, "n_tiles": None, "staging_bytes": send_b + recv_b,
             "volume_ms": volume_ms, "relabel_ms": relabel_ms}
    xinfo = {"gpus": G, "placement": f"ranks in blocks of {P // G}" + ("" if P % G == 0 else " or so"),
             "cross_gpu_elements_identity": int(round(cross0)),
             "cross_gpu_elements_relabeled": int(round(cross1)),
             "send_bytes": send_b, "recv_bytes": recv_b,
             "phase_ms": {k: round(v, 5) for k, v in phase.items()},
             "exchange_gbs_per_gpu": None if phase["exchange"] <= 0 or world == 1
             else round((send_b + recv_b) / (phase["exchange"] * 1e-3) / 1e9, 2)}
    kernel_ms = phase["pack+local"] + phase["unpack"]
    return dict(value=value, ms_per_step=total_ms / args.steps, total_ms=total_ms, per=per,
                launches=launches, clocks=clk, e2e=e2e, plan_s=plan_s, stats=stats,
                nbytes=nbytes, achieved=kernel_bytes / (kernel_ms * 1e-3) / 1e9 if kernel_ms > 0 else 0.0,
                kernel_ms=kernel_ms, kernel_bytes=kernel_bytes,
                peak=peak, peak_kind=peak_kind, traffic=None, probs=probs, phases=None,
                kernels="remap_kernel / remap_small_kernel over the exchange's pack, local and unpack lists",
                exchange=xinfo)


def run_exchange_e2e(args, step, stream, dev, world, nbytes, Bd, Ad, p, A, place, g):
    """End to end for the exchange: every step copies this GPU's rank buffers
    of B (and of A when beta != 0) from pinned host memory, runs the step,
    and copies its rank buffers of A back."""
    import torch
    if args.e2e_steps <= 0:
        return None
    own_a = sorted({int(A.buf[i, j]) for i in range(A.nbr) for j in range(A.nbc)
                    if place[A.owner[i, j]] == g})
    own_b = sorted({int(p.B.buf[i, j]) for i in range(p.B.nbr) for j in range(p.B.nbc)
                    if place[p.B.owner[i, j]] == g})
    hb = {r: torch.empty(Bd.buffer(r).shape, dtype=Bd.arena.dtype, pin_memory=True) for r in own_b}
    ha = {r: torch.empty(Ad.buffer(r).shape, dtype=Ad.arena.dtype, pin_memory=True) for r in own_a}
    for r, t in hb.items():
        t.copy_(Bd.buffer(r))
    for r, t in ha.items():
        t.copy_(Ad.buffer(r))
    torch.cuda.synchronize(dev)

    def e2e_step():
        with torch.cuda.stream(stream):
            for r, t in hb.items():
                Bd.buffer(r).copy_(t, non_blocking=True)
            if p.beta != 0:
                for r, t in ha.items():
                    Ad.buffer(r).copy_(t, non_blocking=True)
            step()
            for r, t in ha.items():
                t.copy_(Ad.buffer(r), non_blocking=True)

    e2e_step()
    torch.cuda.synchronize(dev)
    if world > 1:
        torch.distributed.barrier()
    s2, e2 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s2.record(stream)
    for _ in range(args.e2e_steps):
        e2e_step()
    e2.record(stream)
    torch.cuda.synchronize(dev)
    ms = max_over_ranks(s2.elapsed_time(e2), dev)
    h2d = sum(t.numel() * t.element_size() for t in hb.values())
    if p.beta != 0:
        h2d += sum(t.numel() * t.element_size() for t in ha.values())
    d2h = sum(t.numel() * t.element_size() for t in ha.values())
    return {"value": round(job_throughput(nbytes, 1, args.e2e_steps, ms), 3), "unit": "GB/s",
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "ms_per_step": round(ms / args.e2e_steps, 4), "steps": args.e2e_steps,
            "path": "this GPU's rank buffers copied in from pinned host memory, exchange step, "
                    "A's rank buffers copied out (bytes per GPU)"}


def run_e2e(args, costa, mats, step, stream, dev, world, nbytes):
    """The metric end to end with every step's data in pinned host memory.

    Headline path: the library's layouts point at the pinned host buffers,
    and the kernels read B (and A when beta != 0) and write A over the host
    link inside the timed call.  For reference, the copy path: each step
    copies the inputs host -> device, runs on device storage and copies A
    back."""
    import torch
    from workloads.materialize import block_element_offsets
    hostB = [torch.empty(m[1].arena.shape, dtype=m[1].arena.dtype, pin_memory=True) for m in mats]
    hostA = [torch.empty(m[2].arena.shape, dtype=m[2].arena.dtype, pin_memory=True) for m in mats]
    for (p, Bd, Ad, _, _), hb, ha in zip(mats, hostB, hostA):
        hb.copy_(Bd.arena)
        ha.copy_(Ad.arena)
    torch.cuda.synchronize(dev)

    def host_ptrs(spec, dm, t):
        off = block_element_offsets(spec, dm.starts)
        return (t.data_ptr() + off * t.element_size()).astype("uint64")

    HL = [(costa.costa_layout_from_spec(p.A, p.dtype, host_ptrs(p.A, Ad, ha)),
           costa.costa_layout_from_spec(p.B, p.dtype, host_ptrs(p.B, Bd, hb)))
          for (p, Bd, Ad, _, _), hb, ha in zip(mats, hostB, hostA)]
    probs = [m[0] for m in mats]

    def zero_copy_step():
        if len(HL) > 1:
            costa.costa_transform_batched([h[0] for h in HL], [h[1] for h in HL], [p.op for p in probs],
                                          [p.alpha for p in probs], [p.beta for p in probs], relabel=True,
                                          stream=stream.cuda_stream, mode=args.mode)
        else:
            costa.costa_transform(HL[0][0], HL[0][1], probs[0].op, probs[0].alpha, probs[0].beta,
                                  relabel=True, stream=stream.cuda_stream, mode=args.mode)

    def copy_step():
        with torch.cuda.stream(stream):
            for (p, Bd, Ad, _, _), hb, ha in zip(mats, hostB, hostA):
                Bd.arena.copy_(hb, non_blocking=True)
                if p.beta != 0:
                    Ad.arena.copy_(ha, non_blocking=True)
            step()
            for (p, Bd, Ad, _, _), ha in zip(mats, hostA):
                ha.copy_(Ad.arena, non_blocking=True)

    def timed(fn):
        fn()  # plan for these layouts, outside the timed region
        torch.cuda.synchronize(dev)
        if world > 1:
            torch.distributed.barrier()
        s2, e2 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s2.record(stream)
        for _ in range(args.e2e_steps):
            fn()
        e2.record(stream)
        torch.cuda.synchronize(dev)
        return max_over_ranks(s2.elapsed_time(e2), dev)

    zc_ms = timed(zero_copy_step)
    cp_ms = timed(copy_step)
    for la, lb in HL:
        la.destroy()
        lb.destroy()
    es = esize(probs[0].dtype)
    h2d = sum(p.A.m * p.A.n * es * (2 if p.beta != 0 else 1) for p in probs)
    d2h = sum(p.A.m * p.A.n * es for p in probs)
    cp_h2d = sum(hb.numel() * hb.element_size() for hb in hostB)
    cp_h2d += sum(ha.numel() * ha.element_size() for p, ha in zip(probs, hostA) if p.beta != 0)
    cp_d2h = sum(ha.numel() * ha.element_size() for ha in hostA)
    return {"value": round(job_throughput(nbytes, world, args.e2e_steps, zc_ms), 3), "unit": "GB/s",
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "ms_per_step": round(zc_ms / args.e2e_steps, 4), "steps": args.e2e_steps,
            "path": "storage in pinned host memory: the kernels read B (and A) and write A over the host link",
            "copies": {"value": round(job_throughput(nbytes, world, args.e2e_steps, cp_ms), 3),
                       "ms_per_step": round(cp_ms / args.e2e_steps, 4),
                       "h2d_bytes_per_step": int(cp_h2d), "d2h_bytes_per_step": int(cp_d2h),
                       "path": "cudaMemcpyAsync of whole arenas in, device-storage transform, A copied out"}}


def direct_kernels(costa, mats):
    """Which remap kernels the direct list runs: the tile kernel, and the
    small-tile kernel when small tiles hold at least half of the elements of
    the (batched) list, by the planner's rule (costa_debug_split)."""
    small = total = 0
    tile_kernel = False
    for p, _, _, LA, LB in mats:
        t, pieces, _ = costa.costa_debug_split(LA, LB, p.op)
        if len(pieces):
            small += int((pieces["nx"].astype("int64") * pieces["ny"]).sum())
            tile_kernel |= len(t) > 0
        total += p.A.m * p.A.n
    if len(mats) > 1 and 2 * small < total:
        return "remap_kernel (direct)"
    if small == 0:
        return "remap_kernel (direct)"
    return ("remap_kernel + " if tile_kernel else "") + "remap_small_kernel (direct)"


def message_phases(args, probs, stats, step, stream, dev):
    """Per-phase device time of message mode (pack, local, unpack) from the
    library's phase events, over a separate run of steps after the timed
    region, with the algorithmic bytes of each phase: pack reads and writes
    each remote element once; local and unpack read the source (B or the
    staging), read A when beta != 0 and write A."""
    import torch
    import paper_2106_06601_gb300 as costa
    s = esize(probs[0].dtype)
    reads_a = {p.beta != 0 for p in probs}
    ra = reads_a.pop() if len(reads_a) == 1 else None
    local = stats["local_relabeled"]
    remote = stats["total_volume"] - local
    nbytes = {"pack": 2 * s * remote,
              "local": None if ra is None else (2 + ra) * s * local,
              "unpack": None if ra is None else (2 + ra) * s * remote}
    n = max(10, min(args.steps, 200))
    sums = [0.0, 0.0, 0.0]
    costa.costa_phase_timing(True)
    try:
        with torch.cuda.stream(stream):
            for _ in range(n):
                step()
                ms = costa.costa_phase_times()
                for k in range(3):
                    sums[k] += ms[k]
    finally:
        costa.costa_phase_timing(False)
    torch.cuda.synchronize(dev)
    out = []
    for k, name in enumerate(("pack", "local", "unpack")):
        ms = sums[k] / n
        b = nbytes[name]
        out.append({"phase": name, "ms": round(ms, 5), "bytes": b,
                    "gbs": None if b is None or ms <= 0 else round(b / (ms * 1e-3) / 1e9, 2)})
    return {"steps": n, "phases": out}


def roofline(args, r):
    """Roofline line for the dominant kernel: the direct remap (one launch per
    step for a uniform batch), or in message mode the longest phase."""
    base = {"bound": "hbm", "peak": r["peak"], "unit": "GB/s",
            "peak_source": f"{r['peak_kind']} (MEASURED_PEAKS.json hbm_gbs)"}
    if "exchange" in r:
        ach = r["achieved"]
        base.update({"achieved": round(ach, 2), "frac": round(ach / r["peak"], 4), "traffic": None,
                     "kernel": r["kernels"] + " (per GPU, the collective excluded)",
                     "algorithmic_bytes_per_step": r["kernel_bytes"],
                     "kernel_ms_per_step": round(r["kernel_ms"], 5),
                     "timing": "phase events after the timed region"})
        return base
    ph = r["phases"]
    if ph is not None:
        top = max(ph["phases"], key=lambda x: x["ms"])
        ach = top["gbs"]
        base.update({"achieved": ach, "frac": None if ach is None else round(ach / r["peak"], 4),
                     "traffic": None,
                     "kernel": f"remap_kernel over the {top['phase']} list (message mode)",
                     "algorithmic_bytes_per_launch": top["bytes"],
                     "avg_launch_ms": top["ms"],
                     "timing": f"phase events over {ph['steps']} steps after the timed region"})
        return base
    base.update({"achieved": round(r["achieved"], 2), "frac": round(r["achieved"] / r["peak"], 4),
                 "traffic": r["traffic"], "kernel": r["kernels"],
                 "algorithmic_bytes_per_launch": r["nbytes"],
                 "avg_launch_ms": round(statistics.mean(r["per"]), 5),
                 "median_launch_ms": round(statistics.median(r["per"]), 5),
                 "best_launch_ms": round(min(r["per"]), 5)})
    return base


def cpu_model() -> str:
    """The host CPU's model name, as lscpu or /proc/cpuinfo report it."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except Exception:
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if line.lower().startswith("model name"):
                    return line.split(":", 1)[1].strip()
    except Exception:
        pass
    return platform.machine()


CPU_SAMPLE_MAX_BYTES = 2 * 10 ** 9


def cpu_sample(workload, probs, small):
    """The instance the CPU legs time: the workload's first instance, or,
    when one instance moves more than 2 GB (its host matrices alone take
    minutes to build), the same layouts at reduced size (bench --small:
    c3 at 8192^2, c5 with 16384 of its 131072 rows)."""
    if small or probs[0].algorithmic_bytes() <= CPU_SAMPLE_MAX_BYTES:
        return probs, ""
    red = problems(workload, True)
    p = red[0]
    return red, f"; the same layouts at reduced size: {p.A.m}x{p.A.n}"


def run_cpu_oracle(probs, seconds_target: float, threads: int | None = None, note: str = ""):
    """The oracle, as it stands, on a bounded row slab of the first instance
    (the same layouts and values); returns (GB/s, threads, description, rows,
    seconds per pass, B and A host matrices)."""
    import oracle
    p = probs[0]
    threads = threads or oracle.default_threads()
    Bh = HostMatrix(p.B, p.dtype).fill(p.b_kind, p.seed, p.src_stream)
    Ah = HostMatrix(p.A, p.dtype).fill(p.a_kind, p.seed, p.tgt_stream)
    per_row_bytes = p.A.n * p.esize * (3 if p.beta != 0 else 2)
    # calibrate on a few rows, then size the slab for the target time
    rows = max(1, min(p.A.m, 8))
    t0 = time.perf_counter()
    oracle.transform(p.dtype, p.op, p.alpha, p.beta, p.A, Ah.buffers(), p.B, Bh.buffers(),
                     rows=(0, rows), threads=threads)
    dt = max(time.perf_counter() - t0, 1e-6)
    rows2 = int(min(p.A.m, max(rows, rows * seconds_target / dt)))
    # when the whole instance takes less than the target, repeat it
    reps, done = 0, 0.0
    t0 = time.perf_counter()
    while True:
        oracle.transform(p.dtype, p.op, p.alpha, p.beta, p.A, Ah.buffers(), p.B, Bh.buffers(),
                         rows=(0, rows2), threads=threads)
        reps += 1
        done = time.perf_counter() - t0
        if rows2 < p.A.m or done >= seconds_target:
            break
    dt2 = done / reps
    gbs = rows2 * per_row_bytes / dt2 / 1e9
    desc = (f"rows 0..{rows2} of A ({rows2 * p.A.n} of {p.A.m * p.A.n} elements"
            f"{' of instance 0 of ' + str(len(probs)) if len(probs) > 1 else ''}{note}), "
            f"{reps} pass(es), {done:.1f} s")
    return gbs, threads, desc, rows2, dt2, Bh, Ah


def workload_config(args, workload, probs, world):
    p = probs[0]
    nbytes = algorithmic_bytes(probs)
    text = C.WORKLOAD_TEXT[workload]
    if args.small:
        text = f"{workload} layouts at reduced size ({p.A.m}x{p.A.n} per instance)"
    return {"workload": f"{workload}: {text}",
            "dtype": p.dtype, "op": p.op, "alpha": str(p.alpha), "beta": str(p.beta),
            "P": p.A.nranks, "instances": len(probs), "relabel": True, "mode": args.mode,
            "bytes_per_step_per_gpu": nbytes,
            "l2": f"no flush: inputs larger than L2 ({nbytes / 1e9:.2f} GB moved per step "
                  f"vs {L2_BYTES / 1e6:.0f} MB L2)",
            "parallelism": f"replicas x{world}"}


METRIC = "reshuffle GB/s and % of GB300 HBM peak for A=alpha*op(B)+beta*A, 1 GPU"


def also_list(args):
    if args.also == "none":
        return []
    if args.also == "auto":
        return ["c2", "c3", "c4"] if args.workload == "c5" and not args.small else []
    names = [w for w in args.also.split(",") if w and w != args.workload]
    for w in names:
        if w not in C.CONFIGS and w not in C.EXTRA_WORKLOADS:
            raise SystemExit(f"unknown workload {w}")
    return names


def reference_arm(args, probs):
    """The oracle, as it stands, on the host cores: each step a bounded row
    slab of the headline workload (the same layouts and values)."""
    steps, warmup = max(1, args.steps), max(0, args.warmup)
    # each step sized so that the whole run stays within a few minutes
    per_step = max(0.5, min(10.0, 150.0 / (steps + warmup)))
    import oracle
    threads = oracle.default_threads()
    probs, note = cpu_sample(args.workload, probs, args.small)
    gbs, threads, desc, rows, dt, Bh, Ah = run_cpu_oracle(probs, per_step, note=note)
    p = probs[0]
    per_row_bytes = p.A.n * p.esize * (3 if p.beta != 0 else 2)
    for _ in range(warmup):
        oracle.transform(p.dtype, p.op, p.alpha, p.beta, p.A, Ah.buffers(), p.B,
                         Bh.buffers(), rows=(0, rows), threads=threads)
    t0 = time.perf_counter()
    for _ in range(steps):
        oracle.transform(p.dtype, p.op, p.alpha, p.beta, p.A, Ah.buffers(), p.B,
                         Bh.buffers(), rows=(0, rows), threads=threads)
    dt = time.perf_counter() - t0
    value = rows * per_row_bytes * steps / dt / 1e9
    return {
        "impl": "reference", "metric": METRIC,
        "value": round(value, 4), "unit": "GB/s", "n_gpus": args.gpus, "steps": steps,
        "warmup": warmup, "ms_per_step": round(dt / steps * 1e3, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": p.dtype, "data": "synthetic (seeded counter-based generator)",
        "config": workload_config(args, args.workload, probs, 1),
        "cpu_baseline": {"value": round(value, 4), "unit": "GB/s", "cores": threads,
                         "kind": "oracle", "sample": f"each step: {desc.split(',')[0]}",
                         "cpu_model": cpu_model()},
        "e2e": {"value": round(value, 4), "unit": "GB/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0}}


def measure(args, workload, rank, world, local_rank):
    """One workload on this rank's GPU; on rank 0 the fields of its JSON
    entry (None elsewhere)."""
    import gc
    import torch
    probs = problems(workload, args.small)
    use_x = len(probs) == 1 and (world > 1 or args.exchange)
    r = (run_exchange if use_x else run_gpu)(args, workload, rank, world, local_rank)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cprobs, note = cpu_sample(workload, probs, args.small)
        gbs, threads, desc, _, _, _, _ = run_cpu_oracle(cprobs, args.cpu_seconds, note=note)
        cpu = {"value": round(gbs, 4), "unit": "GB/s", "cores": threads, "kind": "oracle",
               "sample": desc, "cpu_model": cpu_model()}
        if workload in ("c1", "c2"):  # the single-threaded figure as well
            gbs1, _, desc1, _, _, _, _ = run_cpu_oracle(cprobs, min(3.0, args.cpu_seconds), threads=1)
            cpu["single_thread"] = {"value": round(gbs1, 4), "unit": "GB/s", "sample": desc1}
    gc.collect()
    torch.cuda.empty_cache()
    if rank != 0:
        return None
    st = r["stats"]
    out = {
        "value": round(r["value"], 3), "unit": "GB/s",
        "ms_per_step": round(r["ms_per_step"], 5), "dtype": probs[0].dtype,
        "config": workload_config(args, workload, probs, world),
        "elements_per_s": round(sum(p.A.m * p.A.n for p in probs) * world / (r["ms_per_step"] * 1e-3), 1),
        "pct_of_hbm_peak": {"measured": round(100 * r["value"] / world / r["peak"], 2),
                            "nominal_8TBs": round(100 * r["value"] / world / 8000.0, 2)},
        "roofline": roofline(args, r),
        "plan": {"ms": round(r["plan_s"] * 1e3, 2), "volume_ms": round(st["volume_ms"], 3),
                 "relabel_ms": round(st["relabel_ms"], 3), "cells": st["n_cells"],
                 "tiles": st["n_tiles"], "total_volume": st["total_volume"],
                 "local_identity": st["local_identity"],
                 "local_relabeled": st["local_relabeled"],
                 "staging_bytes": st["staging_bytes"]},
        "e2e": r["e2e"], "gpu_launches": r["launches"], "clocks": r["clocks"],
        "cpu_baseline": cpu,
        "scaling": "strong" if use_x else "weak",
    }
    if use_x:
        out["config"]["parallelism"] = f"exchange over {world} GPU(s): pack, NCCL all-to-all-v, unpack"
        out["config"]["mode"] = "exchange"
        out["exchange"] = r["exchange"]
    if r["phases"] is not None:
        out["message_phases"] = r["phases"]
    return out


def main():
    args = parse()
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        if rank != 0:
            return
        print(json.dumps(reference_arm(args, problems(args.workload, args.small))), flush=True)
        return

    import torch
    if world > 1:
        import datetime
        torch.distributed.init_process_group("nccl", device_id=torch.device("cuda", local_rank),
                                             timeout=datetime.timedelta(minutes=3))
    head = measure(args, args.workload, rank, world, local_rank)
    others = {w: measure(args, w, rank, world, local_rank) for w in also_list(args)}
    if rank == 0:
        out = {"metric": METRIC, "value": head.pop("value"), "unit": head.pop("unit"),
               "n_gpus": world, "steps": args.steps, "warmup": max(3, args.warmup),
               "ms_per_step": head.pop("ms_per_step"), "higher_is_better": True,
               "scaling": head.pop("scaling"), "vs_baseline": None, "dtype": head.pop("dtype"),
               "data": "synthetic (seeded counter-based generator, values per the workload)"}
        out.update(head)
        if others:
            for o in others.values():
                o["steps"] = args.steps
            out["per_config"] = others
        print(json.dumps(out), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
