#!/usr/bin/env python3
"""Benchmark of the integer-only relative-positional MHSA on GB300.

One step = one pass of the whole hot path over the encoder workload: 24
stacked attention layers, B = 32 utterances of T = 375 frames (30 s), 8
heads of 128, each layer with its own seeded int8 Q/K/V/P/u/v and its own
dyadic constants (bias vectors, content and position branches, relative
shift, fused requantisation, integer softmax, attn.V and output
requantisation, all in the CUDA kernels behind the C ABI).

Metric: effective TOPS = useful integer ops (6 * dh * T^2 per head and
layer, one multiply-add = 2 ops) / time, plus the attention-only real-time
factor (time / (B * 30 s)).  Inputs stay resident in HBM (1.2 GB per step,
far above the 129 MB L2, so nothing is reused across steps from L2).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Multi-GPU: the path shards with no exchange step (Sec. 3.1 works per
utterance and head, so replicas need no collective on the data path); each
rank runs its own replica of the workload (weak scaling) and `value` sums
the ranks' work over the slowest rank's time.  `--gpus N` with N > 1 and no
WORLD_SIZE in the environment re-launches this script as N ranks under
torch.distributed.run; launched that way already (WORLD_SIZE set), it runs
as one of them.  `--impl reference` times the CPU oracle on the host cores
instead (rank 0 only).
"""
from __future__ import annotations

import argparse
import ctypes
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

WORKLOAD = 3
METRIC = "INT8 rel-pos MHSA effective TOPS & % of roofline; attention RTF at B=32,T=375"
UTT_SECONDS = 30.0          # T = 375 frames at 80 ms
L2_BYTES = 129 * 1024 * 1024
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "fused_kernel_traffic.json")
KERNEL_SRC = os.path.join(ROOT, "paper_2609_30846_gb300", "csrc", "ip_mhsa_kernels.cuh")


def parse_args():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--e2e-steps", type=int, default=3)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=15.0,
                    help="target length of the CPU-baseline sample")
    ap.add_argument("--layers", type=int, default=None,
                    help="profiling only: fewer layers than the workload's 24")
    ap.add_argument("--batch", type=int, default=None,
                    help="profiling only: fewer utterances than the workload's 32")
    ap.add_argument("--no-next-rows", action="store_true",
                    help="skip the projection and feed-forward measurements")
    ap.add_argument("--rows-only", action="store_true",
                    help="profiling: only the projection and feed-forward measurements")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the measurements of the other attention workloads")
    ap.add_argument("--configs-only", type=int, default=None, metavar="W",
                    help="profiling: only the attention workload W (0, 1, 2 or 4), "
                         "--steps launch groups")
    return ap.parse_args()


def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


# ------------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi samples every 200 ms while the timed region runs."""
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(prefix="clocks", suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.QUERY}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)

    def stop(self) -> dict:
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
        rows = []
        if self.path and os.path.exists(self.path):
            with open(self.path) as f:
                for line in f:
                    parts = [x.strip() for x in line.split(",")]
                    if len(parts) >= 9:
                        rows.append(parts)
            os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None
        sm = [num(r[1]) for r in rows if num(r[1]) is not None]
        mx = [num(r[2]) for r in rows if num(r[2]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        loaded = [s for s in sm if mx and s > 0.5 * max(mx)] or sm
        return {"sm_mhz": statistics.median(loaded) if loaded else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(rows)}


# ------------------------------------------------------------------- inputs

def make_layers(n_layers: int, B: int | None = None):
    w = synth.WORKLOADS[WORKLOAD]
    layers = []
    for i in range(n_layers):
        lay = synth.layer(w, i)
        if B is not None and B < w.B:
            lay = synth.Layer(*(np.ascontiguousarray(a[:B]) for a in (lay.q, lay.k, lay.v)),
                              lay.p, lay.u, lay.vb, None, lay.scales)
        layers.append(lay)
    return layers


def useful_ops(B, H, T, dh, layers):
    return 6 * dh * T * T * B * H * layers


def spawn_replicas(nproc: int, argv: list[str], env: dict | None = None) -> int:
    """Runs `python argv...` as `nproc` ranks of one node under
    torch.distributed.run (rendezvous on 127.0.0.1, a free port) and returns
    its exit status; the ranks read RANK / LOCAL_RANK / WORLD_SIZE."""
    import socket
    with socket.socket() as so:
        so.bind(("127.0.0.1", 0))
        port = so.getsockname()[1]
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes", "1",
           "--nproc-per-node", str(nproc), "--master-addr", "127.0.0.1",
           "--master-port", str(port)] + list(argv)
    run_env = dict(os.environ if env is None else env)
    for k in ("WORLD_SIZE", "RANK", "LOCAL_RANK"):
        run_env.pop(k, None)
    return subprocess.run(cmd, env=run_env).returncode


class HostTimer:
    """Wall-clock timer of a timed region (host work, or GPU work followed
    by a synchronisation inside the region)."""

    def start(self):
        self.t0 = time.perf_counter()

    def stop(self) -> float:
        return (time.perf_counter() - self.t0) * 1e3


class EventTimer:
    """CUDA events on the launching stream; stop() waits for the end event."""

    def __init__(self, stream):
        import torch
        self.stream = stream
        self.e0 = torch.cuda.Event(enable_timing=True)
        self.e1 = torch.cuda.Event(enable_timing=True)

    def start(self):
        self.e0.record(self.stream)

    def stop(self) -> float:
        self.e1.record(self.stream)
        self.e1.synchronize()
        return self.e0.elapsed_time(self.e1)


def time_replicas(step, steps: int, dist, timer, sync=lambda: None, device=None):
    """Times `steps` calls of `step` on this rank, bracketed by a barrier and
    `sync` on both sides, and returns (this rank's ms, the slowest rank's
    ms).  Every rank runs its own replica; the job ends with its slowest."""
    if dist is not None:
        dist.barrier()
    sync()
    timer.start()
    for _ in range(steps):
        step()
    ms = timer.stop()
    sync()
    if dist is not None:
        dist.barrier()
    return ms, slowest(dist, ms, device)


def replica_fields(world: int, ops_per_step: float, steps: int, job_ms: float) -> dict:
    """The bench line's job-level fields for `world` replicas of one step of
    `ops_per_step` useful ops each: the value counts every rank's work over
    the slowest rank's time (weak scaling)."""
    return {"value": job_tops(ops_per_step * steps, world, job_ms * 1e-3), "n_gpus": world,
            "ms_per_step": job_ms / steps, "scaling": "weak",
            "parallelism": f"replicas x{world}" if world > 1 else "1 GPU"}


def slowest(dist, x: float, device=None) -> float:
    """Max of a per-rank time over all ranks (x itself without a process
    group): the job ends when its slowest replica ends."""
    if dist is None:
        return x
    import torch
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_tops(ops_per_rank: float, world: int, seconds: float) -> float:
    """Whole-job throughput: every replica does the same work (weak scaling),
    all of it counted, over the slowest rank's time."""
    return ops_per_rank * world / seconds / 1e12


def _counters():
    """The committed ncu counters of the fused kernel, if they were taken on
    the current kernel source (else an empty dict)."""
    if not os.path.exists(TRAFFIC_FILE):
        return {}
    try:
        rec = json.load(open(TRAFFIC_FILE))
        src = hashlib.sha256(open(KERNEL_SRC, "rb").read()).hexdigest()
        return rec if rec.get("kernel_sha256") == src else {}
    except (OSError, ValueError):
        return {}


ROWS_TRAFFIC_FILE = os.path.join(ROOT, "profiles", "next_rows_traffic.json")


def rows_traffic() -> dict:
    """DRAM bytes per launch of the widened rows' kernels from the committed
    ncu record, if every kernel source it names is unchanged (else {})."""
    if not os.path.exists(ROWS_TRAFFIC_FILE):
        return {}
    try:
        rec = json.load(open(ROWS_TRAFFIC_FILE))
        csrc = os.path.join(ROOT, "paper_2609_30846_gb300", "csrc")
        out = {}
        for k, v in rec.get("rows", {}).items():
            # each row names the sources of its kernel and their hashes at capture
            if all(hashlib.sha256(open(os.path.join(csrc, f), "rb").read()).hexdigest() == h
                   for f, h in v["kernel_sha256"].items()):
                out[k] = v["dram_bytes_per_launch"]
        return out
    except (OSError, ValueError, KeyError):
        return {}


def traffic_per_launch():
    """DRAM bytes per fused-kernel launch from the committed ncu summary,
    if it was taken on the current kernel source (else None)."""
    return _counters().get("dram_bytes_per_launch")


def issue_floor(dev, launch_us: float, sm_mhz: float):
    """The ALU bound of the fused kernel: its issued warp instructions per
    launch (committed ncu count on the current source) at one instruction
    per SM sub-partition per cycle (4 per SM) and the SM clock of the run,
    against the measured launch time."""
    inst = _counters().get("smsp_inst_executed_per_launch")
    if not inst or launch_us <= 0 or sm_mhz <= 0:
        return None
    import torch
    nsm = torch.cuda.get_device_properties(dev).multi_processor_count
    floor_us = inst / (nsm * 4 * sm_mhz)
    return {"inst_per_launch": inst, "floor_us": floor_us, "frac": floor_us / launch_us,
            "basis": "issued warp instructions / (SMs x 4 sub-partitions x SM clock)"}


# ------------------------------------------------------------------- oracle arm

def cpu_sample(layers, threads: int, target_s: float):
    """Times the oracle, as it stands, on a bounded sample of the workload:
    the first `nb` utterances of every layer, nb calibrated on one layer."""
    import oracle
    oracle.build()
    oracle.set_threads(threads)
    w = synth.WORKLOADS[WORKLOAD]
    consts = [oracle.layer_constants(l.scales, w.dh) for l in layers]
    q0 = layers[0]
    t = time.perf_counter()
    oracle.relpos_mhsa(np.ascontiguousarray(q0.q[:1]), np.ascontiguousarray(q0.k[:1]),
                       np.ascontiguousarray(q0.v[:1]), q0.p, q0.u, q0.vb, consts[0])
    per_utt_layer = max(time.perf_counter() - t, 1e-4)
    nb = int(max(1, min(w.B, target_s / (per_utt_layer * len(layers)))))
    t = time.perf_counter()
    for lay, c in zip(layers, consts):
        oracle.relpos_mhsa(np.ascontiguousarray(lay.q[:nb]), np.ascontiguousarray(lay.k[:nb]),
                           np.ascontiguousarray(lay.v[:nb]), lay.p, lay.u, lay.vb, c)
    dt = time.perf_counter() - t
    ops = useful_ops(nb, w.H, w.T, w.dh, len(layers))
    # the same oracle on one thread, one 10 s utterance (B=1, T=125)
    w1 = synth.WORKLOADS[1]
    l1 = synth.layer(1, 0)
    c1 = oracle.layer_constants(l1.scales, w1.dh)
    oracle.set_threads(1)
    t1 = time.perf_counter()
    oracle.relpos_mhsa(l1.q, l1.k, l1.v, l1.p, l1.u, l1.vb, c1, l1.lengths)
    dt1 = time.perf_counter() - t1
    oracle.set_threads(threads)
    return {"value": ops / dt / 1e12, "unit": "TOPS", "cores": threads, "kind": "oracle",
            "sample": f"{len(layers)} layers x {nb} of {w.B} utterances (T={w.T}, H={w.H}), "
                      f"{dt:.1f} s, int64 scalar C + OpenMP",
            "one_thread": {"value": useful_ops(w1.B, w1.H, w1.T, w1.dh, 1) / dt1 / 1e12,
                           "unit": "TOPS", "seconds": dt1,
                           "sample": f"one layer, B={w1.B} H={w1.H} T={w1.T}, 1 thread"}}


def run_reference(args):
    world, rank, _ = dist_env()
    if rank != 0:
        return 0
    w = synth.WORKLOADS[WORKLOAD]
    import oracle
    oracle.build()
    threads = os.cpu_count() or 1
    oracle.set_threads(threads)
    layers = make_layers(w.layers, B=1)
    consts = [oracle.layer_constants(l.scales, w.dh) for l in layers]

    def step():
        for lay, c in zip(layers, consts):
            oracle.relpos_mhsa(lay.q, lay.k, lay.v, lay.p, lay.u, lay.vb, c)
    for _ in range(args.warmup):
        step()
    t = time.perf_counter()
    for _ in range(args.steps):
        step()
    dt = time.perf_counter() - t
    ops = useful_ops(1, w.H, w.T, w.dh, w.layers) * args.steps
    value = ops / dt / 1e12
    ms = dt / args.steps * 1e3
    sample = f"per step {w.layers} layers x 1 of {w.B} utterances (T={w.T}, H={w.H})"
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "TOPS", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "int64", "data": "synthetic",
        "config": {"workload": f"{w.name} (sampled: 1 utterance per layer)", "B": 1, "T": w.T,
                   "H": w.H, "dh": w.dh, "layers": w.layers, "l2": "cpu"},
        "rtf": (dt / args.steps) / (1 * UTT_SECONDS),
        "cpu_baseline": {"value": value, "unit": "TOPS", "cores": threads, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "TOPS", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------------------------- next rows

# The projections around the attention of one encoder block (B=32, T=375,
# d=1024): Q/K/V stacked and written head-split, the output projection from
# the attention's row-major output, and the feed-forward pair with the fused
# minimax Swish.
NORM_BUFS = 16

NEXT_ROWS = [
    # name, K, N, groups, x_layout, y_layout, swish
    ("linear_qkv_1024x3072_heads", 1024, 3072, 3, 0, 1, False),
    ("linear_out_1024x1024", 1024, 1024, 1, 0, 0, False),   # reads the attention's row-major O
    ("ffn1_swish_1024x4096", 1024, 4096, 1, 0, 0, True),
    ("ffn2_4096x1024", 4096, 1024, 1, 0, 0, False),
]


# The other attention workloads, each one layer: shapes, distributions and
# (workload 2) key-padding lengths as drawn by synth; launches per timed
# group so that a group lasts well above the event timer's ~2 us tick.
CONFIG_WORKLOADS = (0, 1, 2, 4)
CONFIG_GROUP = {0: 200, 1: 200, 2: 20, 4: 8}


def valid_ops(w, lengths) -> float:
    """Useful ops of one layer of workload w: 6 dh len^2 per (b, h), len the
    utterance's valid length (T without a key-padding mask)."""
    if lengths is None:
        return float(useful_ops(w.B, w.H, w.T, w.dh, 1))
    lens = np.clip(np.asarray(lengths, dtype=np.int64), 0, w.T)
    return float(6 * w.dh * w.H * int(np.sum(lens * lens)))


def measure_configs(dev, peak, pipes, steps: int, cpu: bool, only=None):
    """Per-launch device time of one layer of each other workload: groups of
    CONFIG_GROUP[w] back-to-back launches between one pair of CUDA events on
    the launching stream, L2 flushed before every group (the small workloads
    then read their inputs from HBM in the first launch of a group and from
    L2 after it), median over `steps` groups; useful ops on the valid
    frames; with `cpu`, the oracle timed on the same layer on the host
    cores."""
    import torch
    import paper_2609_30846_gb300 as ip
    stream = torch.cuda.current_stream(dev)
    hstream = ctypes.c_void_p(stream.cuda_stream)
    lib = ip.load()
    flush_w = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    rows = {}
    for wk in (CONFIG_WORKLOADS if only is None else (only,)):
        w = synth.WORKLOADS[wk]
        lay = synth.layer(w, 0)
        c = ip.layer_constants(lay.scales)
        to = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
        d = dict(q=to(lay.q), k=to(lay.k), v=to(lay.v), p=to(lay.p), u=to(lay.u), vb=to(lay.vb))
        lens = None if lay.lengths is None else to(lay.lengths.astype(np.int32))
        out = torch.empty((w.B, w.H, w.T, w.dh), dtype=torch.int8, device=dev)
        ws = torch.zeros(ip.workspace_bytes(w.B, w.H, w.T, w.dh), dtype=torch.uint8, device=dev)
        sm = ip.SoftmaxParams(*c.softmax)
        mult = (ctypes.c_int32 * 3)(*c.multipliers)
        sh = (ctypes.c_int32 * 2)(*c.shifts)
        P = lambda t: None if t is None else ctypes.c_void_p(t.data_ptr())
        args = (P(d["q"]), P(d["k"]), P(d["v"]), P(d["p"]), P(d["u"]), P(d["vb"]), mult, sh,
                ctypes.byref(sm), P(lens), w.B, w.H, w.T, w.dh, P(out), P(ws), ws.numel(), hstream)
        n = CONFIG_GROUP[wk]

        def group():
            for _ in range(n):
                rc = lib.ip_relpos_mhsa_i8(*args)
                if rc != 0:
                    raise ip.IpError("ip_relpos_mhsa_i8", rc, ip.strerror(rc))
        group()
        times = []
        for _ in range(max(steps, 1)):
            flush_w.zero_()
            torch.cuda._sleep(200_000)   # the events and launches queue behind it
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            group()
            e1.record(stream)
            e1.synchronize()
            times.append(e0.elapsed_time(e1) * 1e-3 / n)
        if ip.status(ws, stream) != 0:
            raise SystemExit(f"workload {w.name}: kernel reported an error")
        t = statistics.median(times)
        ops = valid_ops(w, lay.lengths)
        tops = ops / t / 1e12
        bytes_layer = 4 * w.B * w.H * w.T * w.dh + w.H * (2 * w.T - 1) * w.dh
        row = {"workload": w.name, "B": w.B, "H": w.H, "T": w.T, "dh": w.dh,
               "masked": w.masked, "dist": w.dist, "us_per_launch": t * 1e6,
               "value": tops, "unit": "TOPS", "useful_ops": ops,
               "ops_basis": "6 dh len^2 per (b, h), len the valid length" if w.masked
                            else "6 dh T^2 per (b, h)",
               "items": w.B * w.H * ((w.T + 63) // 64),
               "roofline": {"bound": "tensor", "achieved": tops, "peak": peak,
                            "frac": tops / peak,
                            "frac_of_both_integer_pipes": tops / pipes["imma_plus_dp4a"],
                            "hbm_floor_frac": (bytes_layer / (HBM_GBS * 1e9)) / t},
               "timing": f"{n} launches per event pair, L2 flushed before each group, "
                         f"median of {max(steps, 1)} groups",
               "gpu_launches": n * (max(steps, 1) + 1)}
        if cpu:
            import oracle
            oracle.build()
            threads = os.cpu_count() or 1
            oracle.set_threads(threads)
            oc = oracle.layer_constants(lay.scales, w.dh)
            t0 = time.perf_counter()
            oracle.relpos_mhsa(lay.q, lay.k, lay.v, lay.p, lay.u, lay.vb, oc, lay.lengths)
            dt = time.perf_counter() - t0
            row["cpu_baseline"] = {"value": ops / dt / 1e12, "unit": "TOPS", "cores": threads,
                                   "kind": "oracle", "seconds": dt,
                                   "sample": f"the whole layer (B={w.B}, T={w.T})"}
        rows[w.name] = row
        del d, out, ws
    return rows


def measure_next_rows(dev, peak, pipes, steps: int, cpu: bool):
    """Each projection timed alone (CUDA events per launch, L2 flushed before
    every timed launch: a 256 MB write, then a 256 MB read so that no dirty
    line is written back inside the timed launch), useful ops 2 B T K N,
    against the measured throughput of the two integer pipes the linear
    kernel uses together (integer MMA + dp4a; the fraction of the MMA peak
    alone beside it); with `cpu`, the oracle on a bounded sample of frames."""
    both = pipes["imma_plus_dp4a"]
    import torch
    import paper_2609_30846_gb300 as ip
    w0 = synth.WORKLOADS[WORKLOAD]
    B, T = w0.B, w0.T
    flush_w = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    flush_r = torch.ones(256 << 18, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream(dev)

    def flush():
        # write a buffer larger than L2, then read another one, so that the
        # timed launch finds L2 full of clean lines (no write-back inside it);
        # then keep the GPU busy for about 100 us, so that the start event
        # and the timed launches are queued before it goes idle (the host
        # time of issuing them stays out of the measurement)
        flush_w.zero_()
        flush_r.sum()
        torch.cuda._sleep(200_000)

    rows = {}
    traffic = rows_traffic()
    for name, K, N, G, xl, yl, sw in NEXT_ROWS:
        case = synth.linear(B, T, K, N, seed=7000 + K + N + G, groups=G)
        m, s = ip.linear_constants(case.s_x, case.s_w, case.s_y_per_channel())
        x = torch.from_numpy(case.x).to(dev)
        if xl == 1:
            x = x.reshape(B, T, K // 128, 128).permute(0, 2, 1, 3).contiguous()
        w = torch.from_numpy(case.w).to(dev)
        b = torch.from_numpy(case.bias).to(dev)
        md, sd = torch.from_numpy(m).to(dev), torch.from_numpy(s).to(dev)
        ws = torch.zeros(256, dtype=torch.uint8, device=dev)
        swp = ip.swish_params_from_scales(float(case.s_y[0]), 0.9 * float(case.s_y[0])) if sw else None
        if sw:
            out = torch.empty((B, T, N), dtype=torch.int8, device=dev)
            call = lambda: ip.linear_swish_i8(x, w, b, md, sd, swp, out=out, workspace=ws,
                                              stream=stream)
        else:
            ys = (B, T, N) if yl == 0 else (G, B, N // G // 128, T, 128)
            out = torch.empty(ys, dtype=torch.int8, device=dev)
            call = lambda: ip.linear_i8(x, w, b, md, sd, x_layout=xl, y_layout=yl, groups=G,
                                        out=out, workspace=ws, stream=stream)
        for _ in range(3):
            call()
        times = []
        for _ in range(steps):
            flush()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            call()
            e1.record(stream)
            e1.synchronize()
            times.append(e0.elapsed_time(e1) * 1e-3)
        if ip.status(ws, stream) != 0:
            raise SystemExit(f"{name}: kernel reported an error")
        t = statistics.median(times)
        ops = 2.0 * B * T * K * N
        row = {"value": ops / t / 1e12, "unit": "TOPS", "us_per_launch": t * 1e6,
               "shape": {"B": B, "T": T, "K": K, "N": N, "groups": G,
                         "x": "heads" if xl else "rows", "y": "heads" if yl else "rows",
                         "swish": sw},
               "roofline": {"bound": "tensor+dp4a", "achieved": ops / t / 1e12, "peak": both,
                            "unit": "TOPS", "frac": ops / t / 1e12 / both,
                            "frac_of_mma_peak": ops / t / 1e12 / peak,
                            "traffic": traffic.get(name),
                            "peak_source": "measured in this run: integer MMA and dp4a pipes "
                                           "together (ip_probe_int8_mix)"},
               "kernel": "linear_i8_kernel" + ("<swish>" if sw else ""), "gpu_launches": 1}
        if cpu:
            import oracle
            oracle.build()
            def run(frames):
                xs = case.x.reshape(-1, K)[:frames].reshape(1, frames, K)
                t0 = time.perf_counter()
                z = oracle.linear(xs, case.w, case.bias, m, s)
                if sw:
                    oracle.swish(z, oracle.SwishParams(*swp))
                return time.perf_counter() - t0
            # a sample of about one second of oracle work
            frames = 32
            dt = run(frames)
            frames = int(min(B * T, max(32, frames * 1.0 / max(dt, 1e-4))))
            dt = run(frames)
            row["cpu_baseline"] = {"value": 2.0 * frames * K * N / dt / 1e12, "unit": "TOPS",
                                   "cores": os.cpu_count() or 1, "kind": "oracle",
                                   "sample": f"{frames} frames of {B * T}, {dt:.2f} s"}
        rows[name] = row
        del x, w, b, out

    # integer LayerNorm of the frames before the attention (d = 1024).  One
    # launch takes under 20 us, close to the event timer's resolution
    # (about 2 us on this GPU), so a timed group runs NORM_BUFS launches on
    # as many input/output pairs (393 MB, larger than L2) after the flush.
    d = 1024
    nc = synth.norm(B * T, d, seed=7100)
    k = ip.layernorm_constants(nc.s_x, nc.gamma, nc.beta, nc.s_y, nc.eps)
    x0 = torch.from_numpy(nc.x).to(dev)
    xs = [x0] + [x0.clone() for _ in range(NORM_BUFS - 1)]
    outs = [torch.empty_like(x0) for _ in range(NORM_BUFS)]
    Md, Bd, Ed = (torch.from_numpy(a).to(dev) for a in (k.M, k.B, k.E))
    ws = torch.zeros(256, dtype=torch.uint8, device=dev)
    call = lambda i: ip.layernorm_i8(xs[i], Md, Bd, Ed, k.eps_c, out=outs[i], workspace=ws,
                                     stream=stream)
    for i in range(NORM_BUFS):
        call(i)
    times = []
    for _ in range(steps):
        flush()
        torch.cuda._sleep(1_500_000)   # about 0.7 ms: covers the host issue of the group
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for i in range(NORM_BUFS):
            call(i)
        e1.record(stream)
        e1.synchronize()
        times.append(e0.elapsed_time(e1) * 1e-3 / NORM_BUFS)
    if ip.status(ws, stream) != 0:
        raise SystemExit("layernorm: kernel reported an error")
    t = statistics.median(times)
    elems = B * T * d
    ops = NORM_OPS_PER_ELEMENT * elems
    alu_peak = alu_peak_tops(dev)
    row = {"value": elems * 2 / t / 1e9, "unit": "GB/s", "us_per_launch": t * 1e6,
           "shape": {"rows": B * T, "d": d},
           "roofline": {"bound": "alu", "achieved": ops / t / 1e12, "peak": alu_peak,
                        "unit": "Tops/s (int32 lane ops)", "frac": ops / t / 1e12 / alu_peak,
                        "traffic": traffic.get("layernorm_1024"),
                        "hbm_frac": elems * 2 / t / 1e9 / HBM_GBS},
           "kernel": "layernorm_i8_kernel<2>", "gpu_launches": NORM_BUFS,
           "timing": f"{NORM_BUFS} launches on {NORM_BUFS} input/output pairs per event pair"}
    if cpu:
        import oracle
        oracle.build()
        oc = oracle.layernorm_constants(nc.s_x, nc.gamma, nc.beta, nc.s_y, nc.eps)
        n = 512
        t0 = time.perf_counter()
        oracle.layernorm(nc.x[:n], oc)
        dt = time.perf_counter() - t0
        n = int(min(B * T, max(512, n / max(dt, 1e-4))))
        t0 = time.perf_counter()
        oracle.layernorm(nc.x[:n], oc)
        dt = time.perf_counter() - t0
        row["cpu_baseline"] = {"value": n * d * 2 / dt / 1e9, "unit": "GB/s",
                               "cores": os.cpu_count() or 1, "kind": "oracle",
                               "sample": f"{n} frames of {B * T}, {dt:.2f} s"}
    rows["layernorm_1024"] = row
    del xs, outs, x0

    # the ConvBlock's depthwise convolution (K = 9) with the folded
    # BatchNorm onto INT16 and the Swish, on the block's B x T x 1024
    # frames; timed like the LayerNorm (a group of NORM_BUFS launches on as
    # many input/output pairs after the flush)
    C, Kd = 1024, 9
    rng = np.random.default_rng(7200)
    xd0 = torch.from_numpy(rng.integers(-127, 128, size=(B, T, C)).astype(np.int8)).to(dev)
    wd = torch.from_numpy(rng.integers(-127, 128, size=(C, Kd)).astype(np.int8)).to(dev)
    bd = torch.from_numpy(rng.integers(-20000, 20000, size=C).astype(np.int32)).to(dev)
    s_bn = 40.0 / 32767
    md, sd = ip.linear_constants(0.04, rng.uniform(0.001, 0.01, C), np.full(C, s_bn))
    md, sd = torch.from_numpy(md).to(dev), torch.from_numpy(sd).to(dev)
    p16 = ip.swish16_params(s_bn, 5.0 / 127)
    xs = [xd0] + [xd0.clone() for _ in range(NORM_BUFS - 1)]
    outs = [torch.empty_like(xd0) for _ in range(NORM_BUFS)]
    ws = torch.zeros(256, dtype=torch.uint8, device=dev)
    call = lambda i: ip.dwconv_swish_i8(xs[i], wd, bd, md, sd, p16, out=outs[i], workspace=ws,
                                        stream=stream)
    for i in range(NORM_BUFS):
        call(i)
    times = []
    for _ in range(steps):
        flush()
        torch.cuda._sleep(1_500_000)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for i in range(NORM_BUFS):
            call(i)
        e1.record(stream)
        e1.synchronize()
        times.append(e0.elapsed_time(e1) * 1e-3 / NORM_BUFS)
    if ip.status(ws, stream) != 0:
        raise SystemExit("dwconv: kernel reported an error")
    t = statistics.median(times)
    elems = B * T * C
    ops = (2 * Kd + DW_OPS_PER_ELEMENT) * elems
    row = {"value": elems * 2 / t / 1e9, "unit": "GB/s", "us_per_launch": t * 1e6,
           "shape": {"B": B, "T": T, "C": C, "K": Kd},
           "roofline": {"bound": "alu", "achieved": ops / t / 1e12, "peak": alu_peak,
                        "unit": "Tops/s (int32 lane ops)", "frac": ops / t / 1e12 / alu_peak,
                        "traffic": traffic.get("block_dwconv_swish_k9"),
                        "hbm_frac": elems * 2 / t / 1e9 / HBM_GBS},
           "kernel": f"dwconv_swish_x4_kernel<{Kd}>", "gpu_launches": NORM_BUFS,
           "timing": f"{NORM_BUFS} launches on {NORM_BUFS} input/output pairs per event pair"}
    if cpu:
        import oracle
        oracle.build()
        mh, sh = md.cpu().numpy(), sd.cpu().numpy()
        xh, wh, bh = xd0[:1].cpu().numpy(), wd.cpu().numpy(), bd.cpu().numpy()
        t0 = time.perf_counter()
        oracle.swish16(oracle.dwconv(xh, wh, bh, mh, sh), oracle.Swish16Params(*p16))
        dt = time.perf_counter() - t0
        row["cpu_baseline"] = {"value": T * C * 2 / dt / 1e9, "unit": "GB/s",
                               "cores": 1, "kind": "oracle",
                               "sample": f"1 of {B} utterances (T={T}), {dt:.2f} s"}
    rows["dwconv_swish_k9_1024"] = row
    del xs, outs, xd0

    # one whole integer Conformer block (Eqs. 1-5): 15 launches
    import synth.block as sblock
    from paper_2609_30846_gb300.block import GPU_LAUNCHES, ConformerBlock
    case = sblock.conformer_block(B, T, seed=7300)
    blk = ConformerBlock(case, B, T, dev)
    x = torch.from_numpy(case.x).to(dev)
    for _ in range(3):
        blk(x, stream=stream)
    times = []
    for _ in range(steps):
        flush()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        blk(x, stream=stream)
        e1.record(stream)
        e1.synchronize()
        times.append(e0.elapsed_time(e1) * 1e-3)
    if ip.status(blk.ws, stream) != 0:
        raise SystemExit("conformer block: a kernel reported an error")
    t_eager = statistics.median(times)
    # the same fifteen launches captured once into a CUDA graph and replayed
    graph = blk.graph(x)
    times = []
    for _ in range(steps):
        flush()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        graph.replay()
        e1.record(stream)
        e1.synchronize()
        times.append(e0.elapsed_time(e1) * 1e-3)
    torch.cuda.synchronize(dev)
    if ip.status(blk.ws, stream) != 0:
        raise SystemExit("conformer block (graph): a kernel reported an error")
    t = statistics.median(times)
    ops = blk.useful_ops()
    row = {"value": ops / t / 1e12, "unit": "TOPS", "us_per_block": t * 1e6,
           "us_per_block_eager": t_eager * 1e6, "launch": "CUDA graph replay",
           "frames_per_s": B * T / t, "shape": {"B": B, "T": T, "d": 1024, "ff": 4096, "heads": 8},
           "roofline": {"bound": "tensor+dp4a", "achieved": ops / t / 1e12, "peak": both,
                        "unit": "TOPS", "frac": ops / t / 1e12 / both,
                        "frac_of_mma_peak": ops / t / 1e12 / peak, "traffic": None,
                        "traffic_parts": {k: v for k, v in traffic.items() if k.startswith("block_")},
                        "traffic_note": "per kernel in profiles/next_rows_traffic.json; two of "
                                        "the block's fifteen launches (the 1024 -> 1024 "
                                        "projections with the residual) were not captured"},
           "kernel": "15 launches: layernorm x5, linear x8 (2 with Swish, 1 with GLU, 4 with "
                     "the residual addition), relpos_mhsa_fused, dwconv_swish",
           "gpu_launches": GPU_LAUNCHES}
    if cpu:
        import oracle
        from oracle.block import conformer_block as oracle_block
        oracle.build()
        one = sblock.BlockCase(**{**case.__dict__, "x": np.ascontiguousarray(case.x[:1])})
        t0 = time.perf_counter()
        oracle_block(one)
        dt = time.perf_counter() - t0
        row["cpu_baseline"] = {"value": ops / B / dt / 1e12, "unit": "TOPS",
                               "cores": os.cpu_count() or 1, "kind": "oracle",
                               "sample": f"1 of {B} utterances (T={T}), {dt:.1f} s"}
    rows["conformer_block"] = row
    del x, blk, flush_w, flush_r
    return rows


# Integer operations of the LayerNorm per element as the method states them:
# sum and sum of squares (2), centring d q - sum (2), c f with rounding and
# shift (3), M n + B with rounding and shift (3), clamp (2).
NORM_OPS_PER_ELEMENT = 12
# Of the depthwise convolution + INT16 requantisation + Swish, besides the
# K multiply-adds (2 K): bias (1), m acc with rounding and shift (3), clamp
# to INT16 (2), |z| and min(|z|, q_c) - q_c (3), its square and q_one - D^2
# (2), the sign term q_one + sgn(z) L (2), z t (1), m_sw z t with rounding
# and shift (3), clamp (2).
DW_OPS_PER_ELEMENT = 19
def _hbm_gbs() -> float:
    """Measured copy bandwidth of this GPU type (MEASURED_PEAKS.json, written
    by the pool's driver), else the 6.8 TB/s fallback."""
    try:
        return float(json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))["hbm_gbs"])
    except (OSError, ValueError, KeyError):
        return 6800.0


HBM_GBS = _hbm_gbs()


def alu_peak_tops(dev) -> float:
    """One 32-bit integer operation per lane per cycle: SMs x 128 lanes x
    the maximum SM clock."""
    import torch
    props = torch.cuda.get_device_properties(dev)
    try:
        import subprocess as sp
        mhz = float(sp.run(["nvidia-smi", "--query-gpu=clocks.max.sm", "--format=csv,noheader,nounits",
                            f"--id={dev.index or 0}"], capture_output=True, text=True).stdout.split()[0])
    except Exception:
        mhz = 2070.0
    return props.multi_processor_count * 128 * mhz * 1e6 / 1e12


# ------------------------------------------------------------------- GPU arm

def run_ours(args):
    import torch
    import paper_2609_30846_gb300 as ip

    world, rank, local = dist_env()
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU (the attention runs only in CUDA kernels)")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    ip.load()
    if args.rows_only:
        if rank == 0:
            rows = measure_next_rows(dev, ip.int8_mma_peak_tops(), ip.int8_pipe_rates(),
                                     max(args.steps, 1), cpu=False)
            print(json.dumps({"next_rows": rows}), flush=True)
        if dist:
            dist.destroy_process_group()
        return 0

    if args.configs_only is not None:
        if rank == 0:
            rows = measure_configs(dev, ip.int8_mma_peak_tops(), ip.int8_pipe_rates(),
                                   max(args.steps, 1), cpu=False, only=args.configs_only)
            print(json.dumps({"configs": rows}), flush=True)
        if dist:
            dist.destroy_process_group()
        return 0

    w = synth.WORKLOADS[WORKLOAD]
    B, H, T, dh, NL = w.B, w.H, w.T, w.dh, w.layers
    if args.layers:
        NL = min(NL, args.layers)
    if args.batch:
        B = min(B, args.batch)
    reduced = (NL, B) != (w.layers, w.B)
    layers = make_layers(NL, B)
    consts = [ip.layer_constants(l.scales) for l in layers]
    to_dev = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    dl = [dict(q=to_dev(l.q), k=to_dev(l.k), v=to_dev(l.v), p=to_dev(l.p), u=to_dev(l.u),
               vb=to_dev(l.vb), out=torch.empty((B, H, T, dh), dtype=torch.int8, device=dev))
          for l in layers]
    ws = torch.zeros(ip.workspace_bytes(B, H, T, dh), dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)
    lib = ip.load()
    hstream = ctypes.c_void_p(stream.cuda_stream)

    # Pre-marshalled C-ABI arguments of every layer: the timed loop is the
    # bare library calls.
    calls = []
    for d, c in zip(dl, consts):
        sm = ip.SoftmaxParams(*c.softmax)
        mult = (ctypes.c_int32 * 3)(*c.multipliers)
        sh = (ctypes.c_int32 * 2)(*c.shifts)
        ptr = lambda t: ctypes.c_void_p(t.data_ptr())
        calls.append((ptr(d["q"]), ptr(d["k"]), ptr(d["v"]), ptr(d["p"]), ptr(d["u"]), ptr(d["vb"]),
                      mult, sh, ctypes.byref(sm), None, B, H, T, dh, ptr(d["out"]),
                      ctypes.c_void_p(ws.data_ptr()), ws.numel(), hstream, sm))
    fn = lib.ip_relpos_mhsa_i8

    def step():
        for a in calls:
            rc = fn(*a[:-1])
            if rc != 0:
                raise ip.IpError("ip_relpos_mhsa_i8", rc, ip.strerror(rc))

    peak = ip.int8_mma_peak_tops()
    pipes = ip.int8_pipe_rates()
    for _ in range(max(args.warmup, 3)):
        step()
    if ip.status(ws, stream) != 0:
        raise SystemExit("kernel reported a barrier timeout during warm-up")

    # The launches of a step follow one another with nothing between them on
    # the stream (a layer's kernel may then be scheduled while the previous
    # one finishes; it waits for it before touching memory), so the timed
    # region has one pair of events and the per-launch time is its average.
    clocks = ClockSampler(local)
    clocks.start()
    own_ms, total_ms = time_replicas(step, args.steps, dist, EventTimer(stream),
                                     sync=lambda: torch.cuda.synchronize(dev), device=dev)
    clk = clocks.stop()
    if ip.status(ws, stream) != 0:
        raise SystemExit("kernel reported a barrier timeout in the timed region")
    if world > 1:
        print(json.dumps({"rank": rank, "ms": own_ms, "steps": args.steps}), file=sys.stderr,
              flush=True)

    ops_step = useful_ops(B, H, T, dh, NL)
    job = replica_fields(world, ops_step, args.steps, total_ms)
    value = job["value"]
    ms_step = job["ms_per_step"]
    ops_layer = useful_ops(B, H, T, dh, 1)
    avg_layer_ms = total_ms / (args.steps * NL)   # launch gaps included
    achieved = ops_layer / (avg_layer_ms * 1e-3) / 1e12

    # ---- end to end through the host-buffer entry point
    e2e = None
    if args.e2e_steps > 0:
        pin = lambda a: torch.from_numpy(np.ascontiguousarray(a)).pin_memory()
        hl = [dict(q=pin(l.q), k=pin(l.k), v=pin(l.v), p=pin(l.p), u=pin(l.u), vb=pin(l.vb),
                   out=torch.empty((B, H, T, dh), dtype=torch.int8).pin_memory()) for l in layers]
        # three arenas on three streams: a layer's uploads and download
        # (about as long as one kernel at the ~200 GB/s of pinned copies)
        # overlap the kernels of the two layers before it (asynchronous
        # host-buffer calls)
        NA = 3
        arenas = [torch.empty(ip.host_arena_bytes(B, H, T, dh), dtype=torch.uint8, device=dev)
                  for _ in range(NA)]
        streams = [stream] + [torch.cuda.Stream(dev) for _ in range(NA - 1)]

        def e2e_step():
            for li, (h_, c) in enumerate(zip(hl, consts)):
                ip.relpos_mhsa_i8_host(h_["q"], h_["k"], h_["v"], h_["p"], h_["u"], h_["vb"], c,
                                       None, h_["out"], arenas[li % NA], stream=streams[li % NA],
                                       wait=False)
            for j in range(NA):
                if ip.host_status(arenas[j], B, H, T, dh, stream=streams[j]) != 0:
                    raise SystemExit("end-to-end: a kernel reported an error")
        e2e_step()
        torch.cuda.synchronize(dev)
        if dist:
            dist.barrier()
        t = time.perf_counter()
        for _ in range(args.e2e_steps):
            e2e_step()
        torch.cuda.synchronize(dev)
        e2e_s = slowest(dist, time.perf_counter() - t, dev)
        h2d = sum(int(h_[k].numel()) for h_ in hl for k in ("q", "k", "v", "p", "u", "vb"))
        d2h = sum(int(h_["out"].numel()) for h_ in hl)
        e2e = {"value": job_tops(ops_step * args.e2e_steps, world, e2e_s), "unit": "TOPS",
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
               "ms_per_step": e2e_s / args.e2e_steps * 1e3, "steps": args.e2e_steps,
               "streams": NA,
               "note": "the layers are independent problems issued on %d streams: each "
                       "layer's copies and, at the ends of the launches, the kernels of "
                       "neighbouring layers overlap (value times the kernels back to back "
                       "on one stream)" % NA}

    if rank != 0:
        if dist:
            dist.destroy_process_group()
        return 0

    cpu = None
    if world == 1 and not args.no_cpu_baseline:
        cpu = cpu_sample(layers, os.cpu_count() or 1, args.cpu_seconds)
    configs = None
    if not args.no_configs and not reduced:
        configs = measure_configs(dev, peak, pipes, max(args.steps, 5),
                                  cpu=world == 1 and not args.no_cpu_baseline)
    next_rows = None
    if not args.no_next_rows and not reduced:
        next_rows = measure_next_rows(dev, peak, pipes, max(args.steps, 5),
                                      cpu=world == 1 and not args.no_cpu_baseline)

    bytes_layer = 4 * B * H * T * dh + H * (2 * T - 1) * dh + 2 * H * dh
    line = {
        "metric": METRIC, "value": value, "unit": "TOPS", "n_gpus": job["n_gpus"],
        "steps": args.steps, "warmup": max(args.warmup, 3), "ms_per_step": ms_step,
        "higher_is_better": True, "scaling": job["scaling"], "vs_baseline": None, "dtype": "s8xs8->s32 (int32/int64 epilogue)",
        "data": "synthetic",
        "config": {"workload": w.name + (" (REDUCED, profiling only)" if reduced else ""),
                   "B": B, "H": H, "T": T, "dh": dh, "layers": NL,
                   "parallelism": job["parallelism"],
                   "l2": "inputs larger than L2 (%.2f GB per step, L2 129 MB)" % (bytes_layer * NL / 1e9)},
        "rtf": ms_step * 1e-3 / (B * UTT_SECONDS),
        "paper_rtf_npu_full_model": 0.048,
        "roofline": {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TOPS",
                     "frac": achieved / peak, "traffic": traffic_per_launch(),
                     "peak_source": "measured in this run: integer warp MMA (mma.sync m16n8k32 "
                                    "s8) probe, CUDA events; sm_103a has no tcgen05 kind::i8",
                     "hbm_floor_frac": (bytes_layer / (HBM_GBS * 1e9)) / (avg_layer_ms * 1e-3),
                     "alu_floor": issue_floor(dev, avg_layer_ms * 1e3,
                                              (clk or {}).get("sm_mhz") or 2070.0),
                     "integer_pipes_tops": pipes,
                     "frac_of_both_pipes": (achieved / pipes["imma_plus_dp4a"]
                                            if (pipes or {}).get("imma_plus_dp4a") else None),
                     "integer_pipes_note": "measured in this run: the integer MMA pipe and the "
                                           "dp4a pipe alone and together (ip_probe_int8_mix); "
                                           "the fused kernel's contractions use the MMA pipe",
                     "kernel": "relpos_mhsa_fused_kernel (one launch per layer)"},
        "cpu_baseline": cpu,
        "e2e": e2e,
        "gpu_launches": NL * args.steps,
        "clocks": clk,
        "configs": configs,
        "next_rows": next_rows,
    }
    print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()
    return 0


def main():
    args = parse_args()
    if args.gpus > 1 and "WORLD_SIZE" not in os.environ:
        # N replicas were asked for without a launcher: become N ranks
        if args.impl == "ours":
            import torch
            have = torch.cuda.device_count() if torch.cuda.is_available() else 0
            if have < args.gpus:
                raise SystemExit(f"--gpus {args.gpus}: only {have} CUDA device(s) visible")
        return spawn_replicas(args.gpus, [os.path.abspath(__file__)] + sys.argv[1:])
    world, _, _ = dist_env()
    if world != args.gpus and args.gpus > 1:
        raise SystemExit(f"--gpus {args.gpus} but WORLD_SIZE={world}")
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
