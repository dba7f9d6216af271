"""Throughput of the DAMP decode-step state update on GB300.

Workload (one "step" = one decode step of one linear-attention layer over the
whole batch: operand staging, reconstruction, decay, delta read, rank-1
correction, output, requantization and write-back):
    KDA decode, B = 256 request slots, H = 32 heads, d_k = d_v = 128,
    K_hi = 10 FP16 key channels per head, the rest UINT8 + H_32 (G = 32),
    BF16 q/k/v, FP32 gates/beta/o.
Metric: microseconds per step and achieved HBM bandwidth, counted from the
algorithmic bytes of a step (state read + write, q/k/v/beta/gates, o), against
the measured GB300 copy bandwidth.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

Under torchrun every rank runs its own batch (weak scaling, no data exchange);
the step time is the maximum over ranks.  `--impl reference` times the CPU
oracle on a bounded sample of the same workload instead.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import workloads as wl  # noqa: E402

METRIC = "mixed-precision state-update µs/step & achieved HBM TB/s (B=256, vs 8 TB/s peak)"
WORKLOAD = wl.KDA_B256
N_INPUT_SETS = 8
POOLS = 2


def algorithmic_bytes(w: wl.Workload, packed: bool = True) -> int:
    """Bytes a step must move: every state read and written once, operands read once, o written."""
    B, H, Hq, dk, dv, K = w.batch, w.heads, w.qk_heads, w.d_k, w.d_v, w.k_hi
    if packed and w.lo_format == 2:  # row-absmax INT8: one FP32 scale per row
        state = 2 * K * dv + (dk - K) * dv + 4 * (dk - K)
    elif packed:  # codes (8 or 4 bits) + 4 bytes of metadata per 32-group
        bits = 4 if w.lo_format in (3, 4) else 8
        state = 2 * K * dv + (dk - K) * dv * bits // 8 + 4 * (dk - K) * (dv // 32)
    else:
        state = 4 * dk * dv
    esz = 2 if w.in_dtype == "bf16" else 4
    ops = 2 * B * Hq * dk * esz + B * H * dv * esz + B * H * 4 + B * H * (dk if w.kind == "kda" else 1) * 4
    ops += (H * dk) if packed else 0  # the permutation
    return 2 * B * H * state + ops + B * H * dv * 4


# the sources the packed decode step's translation unit compiles (its ncu summary stays
# valid while these are unchanged)
PACKED_STEP_SOURCES = ("decode_packed_kda.cu", "launch_packed.cuh", "decode_packed.cuh", "damp_common.cuh",
                       "damp_internal.h")


def kernel_source_hash() -> str:
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2608_27513_gb300", "csrc")
    for f in PACKED_STEP_SOURCES:
        with open(os.path.join(csrc, f), "rb") as fh:
            h.update(f.encode() + fh.read())
    return h.hexdigest()[:16]


def measured_peaks() -> dict:
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f)
    except OSError:
        return {}


def ncu_traffic(name: str):
    """DRAM bytes per launch from the committed ncu summary, if taken on the current kernel source."""
    path = os.path.join(ROOT, "profiles", f"{name}.txt")
    try:
        kv = {}
        with open(path) as f:
            for line in f:
                if "=" in line and not line.lstrip().startswith("#"):
                    k, v = line.split("=", 1)
                    kv[k.strip()] = v.strip()
        if kv.get("source_hash") == kernel_source_hash():
            return float(kv["dram_bytes_per_launch"])
    except (OSError, KeyError, ValueError):
        pass
    return None


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while the timed region runs."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "50"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        self.out = ""
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.out, _ = self.proc.communicate()

    def summary(self) -> dict:
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in (self.out or "").splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[4:8]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def max_over_ranks(x: float, world: int, device) -> float:
    """The maximum of x over all ranks (the slowest rank sets the step time)."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def make_line(r: dict, steps: int, warmup: int, world: int) -> dict:
    """The bench's JSON line from one rank-0 result (times already maxed over ranks)."""
    w = r["w"]
    bytes_step = algorithmic_bytes(w)
    bytes_fp32 = algorithmic_bytes(w, packed=False)
    ms = r["total_ms"] / steps
    value = world * bytes_step / (ms * 1e-3) / 1e12
    peaks = measured_peaks()
    peak_gbs = peaks.get("hbm_gbs")
    peak_note = "measured" if peak_gbs else "fallback"
    peak_gbs = peak_gbs or 6800.0
    achieved_gbs = bytes_step / (r["launch_ms"] * 1e-3) / 1e9
    return {
        "metric": METRIC, "value": value, "unit": "TB/s", "n_gpus": world, "steps": steps,
        "warmup": warmup, "ms_per_step": ms, "us_per_step": ms * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": workload_config(w, r.get("bits")),
        "clocks": r.get("clocks"),
        "e2e": {"value": world * bytes_step / (r["e2e_ms"] * 1e-3) / 1e12, "unit": "TB/s",
                "us_per_step": r["e2e_ms"] * 1e3, "h2d_bytes_per_step": r["h2d"], "d2h_bytes_per_step": r["d2h"],
                "pipeline": "one packed upload and one read-back per step on a copy stream, overlapping the previous/next step"},
        "gpu_launches": steps,
        "roofline": {"bound": "hbm", "achieved": achieved_gbs, "peak": peak_gbs, "unit": "GB/s",
                     "frac": achieved_gbs / peak_gbs, "peak_source": f"{peak_note} copy bandwidth",
                     "frac_of_8TBs": achieved_gbs / 8000.0,
                     "traffic": ncu_traffic("packed_step_kda_b256"),
                     "kernel": "packed_step_kernel<RL=4,d_k=128,K_hi=10,KDA,H32,BF16>", "algorithmic_bytes": bytes_step},
        "repeats": ({"n": len(r["reps_ms"]), "median_us_per_step": statistics.median(r["reps_ms"]) * 1e3,
                     "min_us_per_step": min(r["reps_ms"]) * 1e3, "max_us_per_step": max(r["reps_ms"]) * 1e3,
                     "note": "five further timed blocks of steps/5 launches each, after 3 warm-up launches"}
                    if r.get("reps_ms") else None),
        "cuda_graph": ({"us_per_step": r["graph_ms"] * 1e3,
                        "note": "the same steps captured in one CUDA graph of 4 launches and replayed"}
                       if r.get("graph_ms") else None),
        "fp32_state_kernel": {"us_per_step": r["fp32_launch_ms"] * 1e3,
                              "achieved_gbs": bytes_fp32 / (r["fp32_launch_ms"] * 1e-3) / 1e9,
                              "bytes_per_step": bytes_fp32,
                              "speedup_of_packed": r["fp32_launch_ms"] / r["launch_ms"]},
        "device": r.get("dev_name"),
        "other_kernels": _side_lines(r.get("side"), peak_gbs, peak_note),
    }


def _side_lines(side, peak_gbs, peak_note):
    """The GDN and row-absmax figures of the same run, each against the same peak."""
    if not side:
        return None
    out = {}
    for k, v in side.items():
        v = dict(v)
        v["frac"] = v["achieved_gbs"] / peak_gbs
        v["frac_of_8TBs"] = v["achieved_gbs"] / 8000.0
        v["peak_source"] = f"{peak_note} copy bandwidth"
        out[k] = v
    return out


def workload_config(w: wl.Workload, bits=None) -> dict:
    world = int(os.environ.get("WORLD_SIZE", "1"))
    return {"workload": w.name, "kind": w.kind, "batch": w.batch, "heads": w.heads, "qk_heads": w.qk_heads,
            "d_k": w.d_k, "d_v": w.d_v, "k_hi": w.k_hi, "lo_format": "uint8 affine G32 + H32",
            "bits_per_value": bits, "in_dtype": w.in_dtype, "bytes_per_step": algorithmic_bytes(w),
            "l2": f"inputs larger than L2: {POOLS} packed state pools of "
                  f"{algorithmic_bytes(w) / 2 / 1e6:.0f} MB each rotated per step (> 129 MB L2)",
            "permutation": "seeded random pi per head (throughput does not depend on which)",
            "timing": "CUDA events around K back-to-back launches on the launching stream; "
                      "roofline.achieved uses the same average launch time",
            "parallelism": f"{world} independent replica(s), one batch per GPU"}


# ------------------------------------------------------------------ GPU arm ---

def gpu_arm(args, rank: int, world: int):
    import torch
    import torch.distributed as dist

    import paper_2608_27513_gb300 as damp

    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", 0)))
    torch.cuda.set_device(dev)
    from paper_2608_27513_gb300 import build
    if rank == 0:
        build.build()
    if world > 1:
        dist.barrier()
    w = WORKLOAD
    L = damp.Layout(w.heads, w.qk_heads, w.d_k, w.d_v, w.k_hi, w.lo_format)
    stream = torch.cuda.current_stream()

    # ---- state: FP32 prefix on the GPU, then the prefill hand-off into the packed cache ----
    prefix_in = wl.torch_step_inputs(w, 16, dev, seed_offset=1000 + rank)
    S = damp.new_fp32_state(L, w.batch, dev)
    o = torch.empty((w.batch, w.heads, w.d_v), device=dev)
    for t in range(w.prefix):
        d = prefix_in[t % len(prefix_in)]
        damp.fp32_kda_decode_step(L, S, d["q"], d["k"], d["v"], d["g"], d["beta"], o=o)
    perm = torch.from_numpy(wl.random_perm(w)).to(dev)
    pools = [damp.new_state(L, w.batch, dev) for _ in range(POOLS)]
    for p in pools:
        damp.quantize_state(L, S, perm, p)
    fp32_pools = [S] + [S.clone() for _ in range(POOLS - 1)]
    inputs = wl.torch_step_inputs(w, N_INPUT_SETS, dev, seed_offset=rank)
    torch.cuda.synchronize()

    def run_packed(i, o_buf):
        d = inputs[i % N_INPUT_SETS]
        damp.kda_decode_step(L, pools[i % POOLS], perm, d["q"], d["k"], d["v"], d["g"], d["beta"], o=o_buf)

    def run_fp32(i, o_buf):
        d = inputs[i % N_INPUT_SETS]
        damp.fp32_kda_decode_step(L, fp32_pools[i % POOLS], d["q"], d["k"], d["v"], d["g"], d["beta"], o=o_buf)

    def timed(fn, steps, warmup, per_launch=False):
        # Back-to-back launches between two CUDA events: an event pair around every
        # launch would add a gap per launch to the timeline being measured.
        for i in range(warmup):
            fn(i, o)
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)] \
            if per_launch else []
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        for i in range(steps):
            if per_launch:
                ev[i][0].record(stream)
            fn(i, o)
            if per_launch:
                ev[i][1].record(stream)
        t1.record(stream)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        total_ms = t0.elapsed_time(t1)
        launch_ms = statistics.mean(a.elapsed_time(b) for a, b in ev) if per_launch else total_ms / steps
        return total_ms, launch_ms

    def max_over_ranks_(x):
        return max_over_ranks(x, world, dev)

    with ClockSampler(dev.index) as clk:
        torch.cuda.nvtx.range_push("timed_packed_step")
        total_ms, launch_ms = timed(run_packed, args.steps, args.warmup)
        torch.cuda.nvtx.range_pop()
    total_ms = max_over_ranks_(total_ms)
    launch_ms = max_over_ranks_(launch_ms)
    if damp.device_status() != 0:
        raise RuntimeError("device status word set during the timed region")
    # five more repetitions of a fifth of the steps each (spread of the measurement)
    reps = []
    for _ in range(5):
        reps.append(max_over_ranks_(timed(run_packed, max(args.steps // 5, 10), 3)[1]))

    # ---- the same steps replayed from a CUDA graph (one graph of 2 * POOLS steps) ----
    gstream = torch.cuda.Stream(dev)
    gstream.wait_stream(stream)
    graph = torch.cuda.CUDAGraph()
    per_graph = 2 * POOLS
    with torch.cuda.graph(graph, stream=gstream):
        for i in range(per_graph):
            run_packed(i, o)
    stream.wait_stream(gstream)
    for _ in range(3):
        graph.replay()
    torch.cuda.synchronize()
    n_graph = max(args.steps // per_graph, 5)
    g0, g1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    g0.record(stream)
    for _ in range(n_graph):
        graph.replay()
    g1.record(stream)
    torch.cuda.synchronize()
    graph_ms = max_over_ranks_(g0.elapsed_time(g1) / (n_graph * per_graph))
    del graph

    # ---- the in-house FP32-state kernel on the same inputs (speedup reference) ----
    fp_steps = max(args.steps // 4, 10)
    fp_total, fp_launch = timed(run_fp32, fp_steps, max(args.warmup, 3))
    fp_launch = max_over_ranks_(fp_launch)

    # ---- end to end through the C ABI from pinned host buffers.  Every step uploads its
    # own inputs and reads its output back; a copy stream overlaps step i+1's upload and
    # step i's read-back with step i's kernel (inputs and outputs double-buffered on the
    # device, events order every reuse). ----
    # A step's operands travel as one packed buffer (each tensor at a 16-B aligned offset),
    # so that every step is one host-to-device and one device-to-host copy.
    copy_stream = torch.cuda.Stream(dev)
    names = list(inputs[0].keys())
    offs, n_bytes = {}, 0
    for k in names:
        offs[k] = n_bytes
        n_bytes += (inputs[0][k].numel() * inputs[0][k].element_size() + 15) // 16 * 16

    def views(buf, like):
        return {k: buf[offs[k]:offs[k] + like[k].numel() * like[k].element_size()].view(like[k].dtype)
                   .view(like[k].shape) for k in names}

    host_buf = [torch.empty(n_bytes, dtype=torch.uint8).pin_memory() for _ in range(2)]
    dev_buf = [torch.empty(n_bytes, dtype=torch.uint8, device=dev) for _ in range(2)]
    for j in range(2):
        for k, t in views(host_buf[j], inputs[0]).items():
            t.copy_(inputs[j][k].cpu())
    dev_in = [views(dev_buf[j], inputs[0]) for j in range(2)]
    o_dev = [torch.empty_like(o) for _ in range(2)]
    o_host = [torch.empty(o.shape, dtype=torch.float32).pin_memory() for _ in range(2)]
    h2d = sum(inputs[0][k].numel() * inputs[0][k].element_size() for k in names)
    d2h = o_host[0].numel() * 4
    up_done = [torch.cuda.Event() for _ in range(2)]
    step_done = [torch.cuda.Event() for _ in range(2)]
    down_done = [torch.cuda.Event() for _ in range(2)]

    def upload(i):
        j = i % 2
        with torch.cuda.stream(copy_stream):
            if i >= 2:
                copy_stream.wait_event(step_done[j])  # step i-2 has read dev_in[j]
            dev_buf[j].copy_(host_buf[j], non_blocking=True)
            up_done[j].record(copy_stream)

    def run_e2e(i):
        j = i % 2
        upload(i + 1)
        stream.wait_event(up_done[j])
        if i >= 2:
            stream.wait_event(down_done[j])  # step i-2's output has been read back
        d = dev_in[j]
        damp.kda_decode_step(L, pools[i % POOLS], perm, d["q"], d["k"], d["v"], d["g"], d["beta"], o=o_dev[j])
        step_done[j].record(stream)
        with torch.cuda.stream(copy_stream):
            copy_stream.wait_event(step_done[j])
            o_host[j].copy_(o_dev[j], non_blocking=True)
            down_done[j].record(copy_stream)

    e2e_steps = max(args.steps // 10, 10)
    e2e_warm = max(args.warmup, 3)
    upload(0)
    for i in range(e2e_warm):
        run_e2e(i)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(e2e_warm, e2e_warm + e2e_steps):
        run_e2e(i)
    stream.wait_event(down_done[(e2e_warm + e2e_steps - 1) % 2])  # the last read-back is inside
    e1.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    e2e_total = max_over_ranks_(e0.elapsed_time(e1))

    # ---- the other kernels the target names, timed the same way on this GPU: GDN B=256
    # K_hi=16 (packed and FP32-state steps) and the row-absmax format on the KDA workload ----
    def side_kernel(ws: wl.Workload, with_fp32: bool):
        Lw = damp.Layout(ws.heads, ws.qk_heads, ws.d_k, ws.d_v, ws.k_hi, ws.lo_format)
        pin = wl.torch_step_inputs(ws, 16, dev, seed_offset=2000 + rank)
        Sw = damp.new_fp32_state(Lw, ws.batch, dev)
        fstep = damp.fp32_kda_decode_step if ws.kind == "kda" else damp.fp32_gdn_decode_step
        pstep = damp.kda_decode_step if ws.kind == "kda" else damp.gdn_decode_step
        for t in range(ws.prefix):
            d = pin[t % len(pin)]
            fstep(Lw, Sw, d["q"], d["k"], d["v"], d["g"], d["beta"], o=o)
        pw = torch.from_numpy(wl.random_perm(ws)).to(dev)
        wpools = [damp.new_state(Lw, ws.batch, dev) for _ in range(POOLS)]
        for p_ in wpools:
            damp.quantize_state(Lw, Sw, pw, p_)
        win = wl.torch_step_inputs(ws, N_INPUT_SETS, dev, seed_offset=3000 + rank)
        wfp = [Sw] + [Sw.clone() for _ in range(POOLS - 1)] if with_fp32 else None
        torch.cuda.synchronize()

        def run_p(i, o_buf):
            d = win[i % N_INPUT_SETS]
            pstep(Lw, wpools[i % POOLS], pw, d["q"], d["k"], d["v"], d["g"], d["beta"], o=o_buf)

        def run_f(i, o_buf):
            d = win[i % N_INPUT_SETS]
            fstep(Lw, wfp[i % POOLS], d["q"], d["k"], d["v"], d["g"], d["beta"], o=o_buf)

        res = {"workload": ws.name, "lo_format": ws.lo_format, "bits_per_value": damp.bits_per_value(Lw)}
        with ClockSampler(dev.index) as clk2:
            _, lp = timed(run_p, args.steps, max(args.warmup, 3))
            lp = max_over_ranks_(lp)
            bytes_w = algorithmic_bytes(ws)
            res.update({"us_per_step": lp * 1e3, "bytes_per_step": bytes_w,
                        "achieved_gbs": bytes_w / (lp * 1e-3) / 1e9})
            if with_fp32:
                _, lf = timed(run_f, max(args.steps // 4, 10), max(args.warmup, 3))
                lf = max_over_ranks_(lf)
                bf = algorithmic_bytes(ws, packed=False)
                res["fp32_state_kernel"] = {"us_per_step": lf * 1e3, "bytes_per_step": bf,
                                            "achieved_gbs": bf / (lf * 1e-3) / 1e9, "speedup_of_packed": lf / lp}
        res["clocks"] = clk2.summary()
        if damp.device_status() != 0:
            raise RuntimeError(f"device status word set during the {ws.name} run")
        del wpools, wfp, Sw
        torch.cuda.empty_cache()
        return res

    side = {"gdn_b256_k16": side_kernel(wl.sweep("gdn", 16), True),
            "kda_b256_k10_row_absmax": side_kernel(w.replace(lo_format=2, name=w.name + "_f2"), False)}
    return {
        "w": w, "total_ms": total_ms, "launch_ms": launch_ms, "fp32_launch_ms": fp_launch, "graph_ms": graph_ms,
        "reps_ms": reps,
        "e2e_ms": e2e_total / e2e_steps, "h2d": h2d, "d2h": d2h, "clocks": clk.summary(),
        "bits": damp.bits_per_value(L), "dev_name": torch.cuda.get_device_name(dev), "side": side,
    }


def _oracle_sample(seconds: float):
    """(state updates done, seconds): the oracle's packed step over 2 slots x H heads of
    the bench workload, repeated for about `seconds` (one host thread)."""
    import numpy as np

    from oracle import core, runs
    w = WORKLOAD
    inp = wl.step_inputs(w, 0, rows=[0, 1])
    units = runs.unit_operands(w, inp)
    n = units["v"].shape[0]
    rng = np.random.default_rng(0)
    perms = np.stack([rng.permutation(w.d_k) for _ in range(n)]).astype(np.uint8)
    S = wl.random_states(1, n, w.d_k, w.d_v, scale=0.3)
    tiers = core.pack_heads(perms, S, w.k_hi, w.lo_format)
    done, t0 = 0, time.perf_counter()
    while time.perf_counter() - t0 < seconds:
        core.mixed_step_heads(perms, *tiers, units["q"], units["k"], units["v"], units["g"], units["beta"],
                              w.k_hi, w.lo_format, w.kind)
        done += n
    return done, time.perf_counter() - t0


def cpu_baseline(seconds: float = 12.0) -> dict:
    """The oracle as it stands, single thread, on a bounded sample of the workload's heads."""
    w = WORKLOAD
    done, el = _oracle_sample(seconds)
    per_unit = algorithmic_bytes(w) / (w.batch * w.heads)
    return {"value": per_unit * done / el / 1e12, "unit": "TB/s", "cores": 1, "kind": "oracle",
            "sample": f"{done} (slot, head) state updates of the KDA B=256 workload "
                      f"({done // (2 * w.heads)} passes over 2 slots x {w.heads} heads), {el:.1f} s, one host thread",
            "us_per_full_step": el / done * w.batch * w.heads * 1e6}


def cpu_baseline_all_cores(seconds: float = 8.0) -> dict:
    """The same sample on every host core at once: one spawned process per core, each
    running the oracle on its own copy (the (slot, head) updates are independent)."""
    import multiprocessing as mp
    w = WORKLOAD
    n = os.cpu_count() or 1
    with mp.get_context("spawn").Pool(n) as pool:
        res = pool.map(_oracle_sample, [seconds] * n)
    done = sum(d for d, _ in res)
    el = max(e for _, e in res)
    per_unit = algorithmic_bytes(w) / (w.batch * w.heads)
    return {"value": per_unit * done / el / 1e12, "unit": "TB/s", "cores": n, "kind": "oracle",
            "sample": f"{done} (slot, head) state updates on {n} processes, {el:.1f} s each",
            "us_per_full_step": el / done * w.batch * w.heads * 1e6}


def reference_arm(args, rank: int, world: int):
    """The CPU oracle on a bounded sample per step (rank 0 only)."""
    import numpy as np

    from oracle import core, runs
    if rank != 0:
        return
    w = WORKLOAD
    inp = wl.step_inputs(w, 0, rows=[0])
    u = runs.unit_operands(w, inp)
    rng = np.random.default_rng(0)
    perms = np.stack([rng.permutation(w.d_k) for _ in range(w.heads)]).astype(np.uint8)
    tiers = core.pack_heads(perms, wl.random_states(2, w.heads, w.d_k, w.d_v, 0.3), w.k_hi, w.lo_format)
    # per-head cost, then heads per step so that warmup + steps fit in about two minutes
    t0 = time.perf_counter()
    core.mixed_step_heads(perms[:4], *(a[:4].copy() for a in tiers), u["q"][:4], u["k"][:4], u["v"][:4],
                          u["g"][:4], u["beta"][:4], w.k_hi, w.lo_format, w.kind)
    per_head = (time.perf_counter() - t0) / 4
    heads = int(max(1, min(w.heads, 120.0 / max(args.steps + args.warmup, 1) / per_head)))
    sl = slice(0, heads)
    sub = [a[sl].copy() for a in tiers]

    def one():
        core.mixed_step_heads(perms[sl], *sub, u["q"][sl], u["k"][sl], u["v"][sl], u["g"][sl], u["beta"][sl],
                              w.k_hi, w.lo_format, w.kind)

    for _ in range(args.warmup):
        one()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        one()
    el = time.perf_counter() - t0
    per_unit = algorithmic_bytes(w) / (w.batch * w.heads)
    value = per_unit * heads * args.steps / el / 1e12
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "TB/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": el / args.steps * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic",
            "config": dict(workload_config(w, 9.0 + 7.0 * w.k_hi / w.d_k),
                           reference="CPU oracle (plain C, FP32, one thread) in place of a reference implementation"),
            "cpu_baseline": {"value": value, "unit": "TB/s", "cores": 1, "kind": "oracle",
                             "sample": f"{heads} of the 8192 (slot, head) updates of a step, per step"},
            "e2e": {"value": value, "unit": "TB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def sweep_arm(steps: int, warmup: int):
    """K_hi sweep at B=256, H=32, d=128 (GDN and KDA) against the FP32-state kernel and
    uniform INT8 (K_hi = 0) with and without H_32: bits/value, bytes and us per step."""
    import torch

    import paper_2608_27513_gb300 as damp
    from paper_2608_27513_gb300 import build
    build.build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    out = []
    for kind in ("gdn", "kda"):
        base = wl.sweep(kind, 0)
        inputs = wl.torch_step_inputs(base, 4, dev)
        S = 0.3 * torch.randn((base.batch, base.heads, base.d_k, base.d_v), device=dev)
        o = torch.empty((base.batch, base.heads, base.d_v), device=dev)

        def timeit(fn, n):
            for i in range(warmup):
                fn(i)
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            for i in range(n):
                fn(i)
            e1.record()
            torch.cuda.synchronize()
            return e0.elapsed_time(e1) / n * 1e3

        L0 = damp.Layout(base.heads, base.qk_heads, base.d_k, base.d_v, 0, 0)
        fp = [S.clone(), S.clone()]
        step32 = damp.fp32_kda_decode_step if kind == "kda" else damp.fp32_gdn_decode_step
        us = timeit(lambda i: step32(L0, fp[i % 2], inputs[i % 4]["q"], inputs[i % 4]["k"], inputs[i % 4]["v"],
                                     inputs[i % 4]["g"], inputs[i % 4]["beta"], o=o), max(steps // 4, 10))
        nb = algorithmic_bytes(base, packed=False)
        out.append({"kind": kind, "format": "fp32 state", "k_hi": None, "bits_per_value": 32.0,
                    "bytes_per_step": nb, "us_per_step": us, "tb_s": nb / us / 1e6})
        del fp
        perm = torch.from_numpy(wl.random_perm(base)).to(dev)
        points = [(0, 1, "uniform int8 (no H32)"), (0, 0, "uniform int8 + H32")] + \
                 [(k, 0, "damp fp16 + int8 + H32") for k in wl.SWEEP_K_HI if k > 0] + \
                 [(0, 2, "uniform int8 row-absmax"), (16, 2, "fp16 + int8 row-absmax"),
                  (0, 3, "uniform int4 + H32"), (0, 4, "uniform int4 (no H32)"), (0, 5, "uniform fp8 e4m3"),
                  (16, 3, "fp16 + int4 + H32")]
        for k, fmt, name in points:
            w = wl.sweep(kind, k, fmt)
            L = damp.Layout(w.heads, w.qk_heads, w.d_k, w.d_v, k, fmt)
            pools = [damp.new_state(L, w.batch, dev) for _ in range(2)]
            for pl in pools:
                damp.quantize_state(L, S, perm, pl)
            if k == 0:
                step = damp.u8_kda_decode_step if kind == "kda" else damp.u8_gdn_decode_step
            else:
                step = damp.kda_decode_step if kind == "kda" else damp.gdn_decode_step
            us = timeit(lambda i: step(L, pools[i % 2], perm, inputs[i % 4]["q"], inputs[i % 4]["k"],
                                       inputs[i % 4]["v"], inputs[i % 4]["g"], inputs[i % 4]["beta"], o=o), steps)
            nb = algorithmic_bytes(w)
            out.append({"kind": kind, "format": name, "k_hi": k, "bits_per_value": damp.bits_per_value(L),
                        "bytes_per_step": nb, "us_per_step": us, "tb_s": nb / us / 1e6})
            del pools
    if damp.device_status() != 0:
        raise RuntimeError("device status word set during the sweep")
    for row in out:
        print(json.dumps(row), flush=True)


def prefill_arm(steps: int, warmup: int, T: int = 64, lo_format: int = 0, kinds=("kda", "gdn"), batch: int = 256):
    """Prefill chunks (App. A.5 prefill path) at B = 256 (or `batch`), H = 32, d = 128: one
    launch per chunk of T tokens per slot.  Chunks of 32+ tokens on the affine tiers run
    the chunkwise closed form on the tensor cores; others the per-token FP32 recurrence
    with each tile's state on chip.  Reported against the FP32 FMA peak (SMs x 4
    sub-partitions x 32 lanes x 2 flops x SM clock) with the per-token form's FLOPs."""
    import torch

    import paper_2608_27513_gb300 as damp
    from paper_2608_27513_gb300 import build
    build.build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    out = []
    ws = {"kda": wl.KDA_B256.replace(lo_format=lo_format), "gdn": wl.sweep("gdn", 16, lo_format)}
    for w in (ws[k].replace(batch=batch) for k in kinds):
        L = damp.Layout(w.heads, w.qk_heads, w.d_k, w.d_v, w.k_hi, w.lo_format)
        per_t = wl.torch_step_inputs(w, T, dev)
        chunk = {key: torch.stack([d[key] for d in per_t], dim=1).contiguous() for key in per_t[0]}
        del per_t
        perm = torch.from_numpy(wl.random_perm(w)).to(dev)
        S = 0.3 * torch.randn((w.batch, w.heads, w.d_k, w.d_v), device=dev)
        pools = [damp.new_state(L, w.batch, dev) for _ in range(2)]
        for pl in pools:
            damp.quantize_state(L, S, perm, pl)
        del S
        o = torch.empty((w.batch, T, w.heads, w.d_v), device=dev)
        fn = damp.kda_prefill_chunk if w.kind == "kda" else damp.gdn_prefill_chunk

        def run(i):
            fn(L, pools[i % 2], perm, chunk["q"], chunk["k"], chunk["v"], chunk["g"], chunk["beta"], o=o)

        for i in range(warmup):
            run(i)
        torch.cuda.synchronize()
        n = max(steps // 100, 5)
        with ClockSampler(dev.index) as clk:
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            for i in range(n):
                run(i)
            e1.record()
            torch.cuda.synchronize()
        us = e0.elapsed_time(e1) / n * 1e3
        flops = 7.0 * w.d_k * w.d_v * w.batch * w.heads * T  # decay 1, r 2, p 2, update 2 per state element
        clocks = clk.summary()
        mhz = (clocks or {}).get("sm_mhz") or 2070.0
        peak = sms * 4 * 32 * 2 * mhz * 1e6
        esz = 2 if w.in_dtype == "bf16" else 4
        hbm = (2 * w.batch * w.heads * damp.slot_bytes(L) // w.heads
               + w.batch * T * (2 * w.qk_heads * w.d_k * esz + w.heads * w.d_v * (esz + 4)
                                + w.heads * 4 * ((w.d_k if w.kind == "kda" else 1) + 1)))
        # which chunk kernel the library runs for this call (the dispatch rule of launch_prefill.cuh)
        tc = w.lo_format in (0, 1, 3, 4) and T >= 32 and w.d_k == w.d_v == 128 and w.in_dtype == "bf16"
        kernel = (f"prefill_tc_{w.kind}_kernel (chunkwise closed form on the tensor cores)" if tc else
                  "prefill_cg_kernel (per-token FP32 recurrence)" if w.lo_format in (0, 1) and T >= 32 else
                  "prefill_chunk_kernel (per-token FP32 recurrence)")
        out.append({"mode": "prefill_chunk", "kind": w.kind, "workload": w.name, "batch": w.batch,
                    "lo_format": w.lo_format, "chunk_tokens": T, "kernel": kernel,
                    "us_per_chunk": us, "tokens_per_s": w.batch * T / (us * 1e-6),
                    # the per-token form's FLOPs against the FP32 FMA peak: for the tensor-core
                    # kernel an equivalent rate (its work is tensor-core products plus the solve)
                    "roofline": {"bound": "fma", "achieved": flops / (us * 1e-6) / 1e12, "peak": peak / 1e12,
                                 "unit": "TFLOP/s", "frac": flops / (us * 1e-6) / peak,
                                 "peak_source": f"FP32 FMA: {sms} SMs x 128 lanes x 2 flops x {mhz:.0f} MHz",
                                 "flops": "7 per state element per token (per-token form)"},
                    "hbm_gbs": hbm / (us * 1e-6) / 1e9, "clocks": clocks})
        del pools, chunk, o
    if damp.device_status() != 0:
        raise RuntimeError("device status word set during the prefill runs")
    for row in out:
        print(json.dumps(row), flush=True)


def multitoken_arm(steps: int, warmup: int, tokens=(1, 2, 4, 8, 16)):
    """Fused multi-token steps at the decode workload (KDA, B = 256, H = 32, d = 128,
    K_hi = 10): T tokens per request slot in one launch of the chunk kernel (the state is
    read and requantized once for the T tokens), against T single-token launches of the
    packed decode step on the same pools.  Reports us per launch and per token."""
    import torch

    import paper_2608_27513_gb300 as damp
    from paper_2608_27513_gb300 import build
    build.build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    w = wl.KDA_B256
    L = damp.Layout(w.heads, w.qk_heads, w.d_k, w.d_v, w.k_hi, w.lo_format)
    perm = torch.from_numpy(wl.random_perm(w)).to(dev)
    S = 0.3 * torch.randn((w.batch, w.heads, w.d_k, w.d_v), device=dev)
    pools = [damp.new_state(L, w.batch, dev) for _ in range(2)]
    for pl in pools:
        damp.quantize_state(L, S, perm, pl)
    del S
    per_t = wl.torch_step_inputs(w, max(tokens), dev)

    def timeit(fn, n):
        for i in range(warmup):
            fn(i)
        torch.cuda.synchronize()
        with ClockSampler(dev.index) as clk:
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            for i in range(n):
                fn(i)
            e1.record()
            torch.cuda.synchronize()
        return e0.elapsed_time(e1) / n * 1e3, clk.summary()

    o1 = torch.empty((w.batch, w.heads, w.d_v), device=dev)

    def step(i):
        d = per_t[i % len(per_t)]
        damp.kda_decode_step(L, pools[i % 2], perm, d["q"], d["k"], d["v"], d["g"], d["beta"], o=o1)

    us_step, _ = timeit(step, max(steps, 200))
    out = []
    esz = 2 if w.in_dtype == "bf16" else 4
    state = 2 * w.batch * damp.slot_bytes(L)
    for T in tokens:
        chunk = {key: torch.stack([d[key] for d in per_t[:T]], dim=1).contiguous() for key in per_t[0]}
        o = torch.empty((w.batch, T, w.heads, w.d_v), device=dev)

        def run(i):
            damp.kda_prefill_chunk(L, pools[i % 2], perm, chunk["q"], chunk["k"], chunk["v"], chunk["g"],
                                   chunk["beta"], o=o)

        us, clocks = timeit(run, max(steps // (4 * T), 20))
        ops = w.batch * T * (2 * w.qk_heads * w.d_k * esz + w.heads * w.d_v * (esz + 4)
                             + w.heads * 4 * (w.d_k + 1))
        out.append({"mode": "multi_token_step", "kind": w.kind, "workload": w.name, "tokens": T,
                    "us_per_launch": us, "us_per_token": us / T, "tokens_per_s": w.batch * T / (us * 1e-6),
                    "single_token_steps_us": us_step * T, "speedup_vs_single_steps": us_step * T / us,
                    "algorithmic_bytes": state + ops, "hbm_gbs": (state + ops) / (us * 1e-6) / 1e9,
                    "clocks": clocks})
        del chunk, o
    if damp.device_status() != 0:
        raise RuntimeError("device status word set during the multi-token runs")
    for row in out:
        print(json.dumps(row), flush=True)


def calibrate_arm(steps: int, warmup: int, n_docs: int = 32, n_tokens: int = 256):
    """Calibration run (Algorithm 1, App. A.2) on the GPU for one layer of H = 32 heads,
    d = 128: FP32 trajectories of n_docs documents over n_tokens tokens, error energy of
    the states every 8 tokens, mean log-decay, selection.  Reports the whole run and the
    error-energy pass alone (HBM-bound: it reads the sampled states once)."""
    import torch

    import paper_2608_27513_gb300 as damp
    from paper_2608_27513_gb300 import build, calibration
    build.build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    peak = measured_peaks().get("hbm_gbs") or 6800.0
    out = []
    for w in (wl.stack_layer(1, 16), wl.stack_layer(0, 16)):
        w = w.replace(batch=n_docs)
        L = damp.Layout(w.heads, w.qk_heads, w.d_k, w.d_v, w.k_hi, w.lo_format)
        inputs = wl.torch_step_inputs(w, n_tokens, dev)
        calibration.calibrate(L, w.kind, inputs[:16])  # warm-up
        # the documents' tokens as stacked [T, B, ...] tensors, as a calibration set is stored
        inputs = {n: torch.stack([d[n] for d in inputs]) for n in ("q", "k", "v", "g", "beta")}
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        C, perm = calibration.calibrate(L, w.kind, inputs)
        e1.record()
        torch.cuda.synchronize()
        run_ms = e0.elapsed_time(e1)
        # the same run captured in one CUDA graph and replayed: the GPU time of the run's
        # launches without the host issuing them one by one
        gs = torch.cuda.Stream(dev)
        gs.wait_stream(torch.cuda.current_stream())
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=gs):
            calibration.calibrate(L, w.kind, inputs, stream=gs)
        torch.cuda.current_stream().wait_stream(gs)
        graph.replay()
        torch.cuda.synchronize()
        e0.record()
        graph.replay()
        e1.record()
        torch.cuda.synchronize()
        graph_ms = e0.elapsed_time(e1)
        del graph
        # the error-energy pass alone, on 3 x n_docs sampled states (201 MB at 96 x 32 x 128 x 128
        # FP32: larger than L2, so every call reads its states from HBM)
        ee_docs = 3 * n_docs
        S = 0.3 * torch.randn((ee_docs, w.heads, w.d_k, w.d_v), device=dev)
        E = torch.zeros((w.heads, w.d_k), device=dev)
        for _ in range(max(warmup, 3)):
            damp.calib_error_energy(L, S, E)
        n = max(steps // 20, 10)
        torch.cuda.synchronize()
        e0.record()
        for _ in range(n):
            damp.calib_error_energy(L, S, E)
        e1.record()
        torch.cuda.synchronize()
        ee_us = e0.elapsed_time(e1) / n * 1e3
        gbs = S.numel() * 4 / (ee_us * 1e-6) / 1e9
        out.append({"mode": "calibration", "kind": w.kind, "docs": n_docs, "tokens": n_tokens, "heads": w.heads,
                    "d": w.d_k, "k_hi": w.k_hi, "run_ms": run_ms, "run_ms_cuda_graph_replay": graph_ms,
                    "error_energy_batch": ee_docs, "error_energy_us_per_call": ee_us,
                    "error_energy_roofline": {"bound": "hbm", "achieved": gbs, "peak": peak, "unit": "GB/s",
                                              "frac": gbs / peak, "bytes_per_call": S.numel() * 4}})
        del inputs, S
    if damp.device_status() != 0:
        raise RuntimeError("device status word set during the calibration runs")
    for row in out:
        print(json.dumps(row), flush=True)


def drift_arm(layers: int = 30, steps: int = 1024, every: int = 64):
    """Free-running drift of the 30-layer stack (15 GDN + 15 KDA, alternating; B = 256,
    H = 32, d = 128): per layer, pi from a GPU calibration run (32 documents x 256
    tokens), a 256-token FP32 prefix, then `steps` decode steps of the FP32 state, of
    DAMP (K_hi = 16, calibrated pi) and of uniform INT8 + H_32 (K_hi = 0) on the same
    inputs.  Drift = held-out trajectory RRMSE (App. E): output RRMSE over every step,
    state RRMSE over the states every `every` steps."""
    import torch

    import paper_2608_27513_gb300 as damp
    from paper_2608_27513_gb300 import build, calibration
    build.build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    rows = []
    block = 64
    for layer in range(layers):
        w = wl.stack_layer(layer, 16)
        Ld = damp.Layout(w.heads, w.qk_heads, w.d_k, w.d_v, 16, 0)
        Lu = damp.Layout(w.heads, w.qk_heads, w.d_k, w.d_v, 0, 0)
        calib = wl.torch_step_inputs(w.replace(batch=32), 256, dev, seed_offset=7_000_000)
        _, perm_d = calibration.calibrate(Ld, w.kind, calib)
        del calib
        perm_u = torch.arange(w.d_k, dtype=torch.uint8, device=dev).repeat(w.heads, 1)
        fp32 = damp.fp32_kda_decode_step if w.kind == "kda" else damp.fp32_gdn_decode_step
        packed = damp.kda_decode_step if w.kind == "kda" else damp.gdn_decode_step
        S = damp.new_fp32_state(Ld, w.batch, dev)
        o = torch.empty((w.batch, w.heads, w.d_v), device=dev)
        for t0 in range(0, w.prefix, block):
            for d in wl.torch_step_inputs(w, min(block, w.prefix - t0), dev, seed_offset=1_000_000 + t0):
                fp32(Ld, S, d["q"], d["k"], d["v"], d["g"], d["beta"], o=o)
        st_d = damp.new_state(Ld, w.batch, dev)
        st_u = damp.new_state(Lu, w.batch, dev)
        damp.quantize_state(Ld, S, perm_d, st_d)
        damp.quantize_state(Lu, S, perm_u, st_u)
        acc = torch.zeros(6, dtype=torch.float64, device=dev)  # o: err_d, err_u, ref; state: err_d, err_u, ref
        od = torch.empty_like(o)
        ou = torch.empty_like(o)
        for t0 in range(0, steps, block):
            for i, d in enumerate(wl.torch_step_inputs(w, min(block, steps - t0), dev, seed_offset=2_000_000 + t0)):
                fp32(Ld, S, d["q"], d["k"], d["v"], d["g"], d["beta"], o=o)
                packed(Ld, st_d, perm_d, d["q"], d["k"], d["v"], d["g"], d["beta"], o=od)
                packed(Lu, st_u, perm_u, d["q"], d["k"], d["v"], d["g"], d["beta"], o=ou)
                acc[0] += ((od - o).double() ** 2).sum()
                acc[1] += ((ou - o).double() ** 2).sum()
                acc[2] += (o.double() ** 2).sum()
                if (t0 + i + 1) % every == 0:
                    Sd = damp.dequantize_state(Ld, st_d, perm_d)
                    acc[3] += ((Sd - S).double() ** 2).sum()
                    del Sd
                    Su = damp.dequantize_state(Lu, st_u, perm_u)
                    acc[4] += ((Su - S).double() ** 2).sum()
                    del Su
                    acc[5] += (S.double() ** 2).sum()
        a = acc.cpu().numpy()
        rows.append({"mode": "drift", "layer": layer, "kind": w.kind, "steps": steps,
                     "damp_k16": {"o_rrmse": float(np.sqrt(a[0] / a[2])), "state_rrmse": float(np.sqrt(a[3] / a[5]))},
                     "uniform_int8_h32": {"o_rrmse": float(np.sqrt(a[1] / a[2])),
                                          "state_rrmse": float(np.sqrt(a[4] / a[5]))},
                     "bits_per_value": {"damp_k16": damp.bits_per_value(Ld), "uniform": damp.bits_per_value(Lu)}})
        print(json.dumps(rows[-1]), flush=True)
        del S, st_d, st_u, o, od, ou
        torch.cuda.empty_cache()
    if damp.device_status() != 0:
        raise RuntimeError("device status word set during the drift run")


def tiered_arm(steps: int = 512, every: int = 64, batch: int = 64, timing_steps: int = 1000):
    """Decay-tiered per-head K_hi (App. E, head-budget ablation) on a GDN layer (H = 32,
    d = 128, B = 64): the even heads decay fast and the odd heads slowly (gate logit
    bias +1 / -3, median alpha ~0.23 / ~0.95).  Allocations common 16/16 and
    K_fast/K_slow in {12/20, 8/24, 4/28} (mean 16, the same bytes), each a pair of head
    groups with pi from a GPU calibration per group; then `steps` decode steps from a
    256-step FP32 prefix.  Drift = held-out RRMSE against the FP32 trajectory (output every
    step, state every `every` steps).  Also times one layer step at B = 256 as one launch
    (common) and as two group launches (4/28)."""
    import torch

    import paper_2608_27513_gb300 as damp
    from paper_2608_27513_gb300 import build, calibration
    build.build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    w = wl.sweep("gdn", 16).replace(batch=batch)
    H = w.heads
    fast = [h % 2 == 0 for h in range(H)]
    bias = [1.0 if f else -3.0 for f in fast]
    allocs = [(16, 16), (12, 20), (8, 24), (4, 28)]
    calib = wl.torch_step_inputs(w.replace(batch=32), 256, dev, seed_offset=7_000_000, gate_bias=bias)
    setups = []
    for kf, ks in allocs:
        groups = damp.head_groups([kf if f else ks for f in fast], w.qk_heads, w.d_k, w.d_v, device=dev)
        sel = calibration.calibrate_groups(groups, "gdn", calib)
        setups.append([(L, hs, pi) for (L, hs), (_, pi) in zip(groups, sel)])
    del calib
    Lf = damp.Layout(H, w.qk_heads, w.d_k, w.d_v, 0, 0)
    S = damp.new_fp32_state(Lf, w.batch, dev)
    o = torch.empty((w.batch, H, w.d_v), device=dev)
    for d in wl.torch_step_inputs(w, 256, dev, seed_offset=1_000_000, gate_bias=bias):
        damp.fp32_gdn_decode_step(Lf, S, d["q"], d["k"], d["v"], d["g"], d["beta"], o=o)
    pools = [[damp.new_state(L, w.batch, dev) for L, _, _ in gs] for gs in setups]
    for gs, ps in zip(setups, pools):
        for (L, hs, pi), pl in zip(gs, ps):
            damp.quantize_state(L, S, pi, pl)
    acc = torch.zeros((len(allocs), 4), dtype=torch.float64, device=dev)  # o err, o ref, state err, state ref
    oa = torch.empty_like(o)
    for t0 in range(0, steps, 64):
        for i, d in enumerate(wl.torch_step_inputs(w, min(64, steps - t0), dev, seed_offset=2_000_000 + t0,
                                                   gate_bias=bias)):
            damp.fp32_gdn_decode_step(Lf, S, d["q"], d["k"], d["v"], d["g"], d["beta"], o=o)
            sample = (t0 + i + 1) % every == 0
            for a, (gs, ps) in enumerate(zip(setups, pools)):
                for (L, hs, pi), pl in zip(gs, ps):
                    damp.gdn_decode_step(L, pl, pi, d["q"], d["k"], d["v"], d["g"], d["beta"], o=oa)
                acc[a, 0] += ((oa - o).double() ** 2).sum()
                acc[a, 1] += (o.double() ** 2).sum()
                if sample:
                    Sa = torch.zeros_like(S)
                    for (L, hs, pi), pl in zip(gs, ps):
                        damp.dequantize_state(L, pl, pi, S=Sa)
                    acc[a, 2] += ((Sa - S).double() ** 2).sum()
                    acc[a, 3] += (S.double() ** 2).sum()
                    del Sa
    a = acc.cpu().numpy()
    rows = []
    for i, (kf, ks) in enumerate(allocs):
        rows.append({"mode": "decay_tiered", "kind": "gdn", "batch": w.batch, "steps": steps, "k_fast": kf,
                     "k_slow": ks, "state_rrmse": float(np.sqrt(a[i, 2] / a[i, 3])),
                     "o_rrmse": float(np.sqrt(a[i, 0] / a[i, 1])),
                     "bytes_per_slot": int(sum(damp.slot_bytes(L) for L, _, _ in setups[i]))})
    # one layer step at B = 256: the common layout (one launch) and the 4/28 groups (two launches)
    wb = w.replace(batch=256)
    inputs = wl.torch_step_inputs(wb, 4, dev, gate_bias=bias)
    Lc = damp.Layout(H, w.qk_heads, w.d_k, w.d_v, 16, 0)
    pc = [damp.new_state(Lc, 256, dev) for _ in range(2)]
    tiered = setups[-1]
    pt = [[damp.new_state(L, 256, dev) for L, _, _ in tiered] for _ in range(2)]
    perm_c = setups[0][0][2]
    o2 = torch.empty((256, H, w.d_v), device=dev)

    def common(i):
        d = inputs[i % 4]
        damp.gdn_decode_step(Lc, pc[i % 2], perm_c, d["q"], d["k"], d["v"], d["g"], d["beta"], o=o2)

    def groups(i):
        d = inputs[i % 4]
        for (L, hs, pi), pl in zip(tiered, pt[i % 2]):
            damp.gdn_decode_step(L, pl, pi, d["q"], d["k"], d["v"], d["g"], d["beta"], o=o2)

    def one_launch(setup):
        pools2 = [[damp.new_state(L, 256, dev) for L, _, _ in setup] for _ in range(2)]

        def run(i):
            d = inputs[i % 4]
            damp.gdn_decode_step_groups([(L, pl, pi) for (L, _, pi), pl in zip(setup, pools2[i % 2])],
                                        d["q"], d["k"], d["v"], d["g"], d["beta"], o=o2)
        return run

    timing = {}
    for name, fn in (("common_k16_one_launch", common), ("tiered_4_28_two_launches", groups),
                     ("tiered_12_20_one_launch", one_launch(setups[1])), ("tiered_8_24_one_launch", one_launch(setups[2])),
                     ("tiered_4_28_one_launch", one_launch(setups[3]))):
        for i in range(20):
            fn(i)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for i in range(timing_steps):
            fn(i)
        e1.record()
        torch.cuda.synchronize()
        timing[name] = e0.elapsed_time(e1) / timing_steps * 1e3
    rows.append({"mode": "decay_tiered_step_time", "kind": "gdn", "batch": 256, "us_per_step": timing})
    if damp.device_status() != 0:
        raise RuntimeError("device status word set during the decay-tiered run")
    for r in rows:
        print(json.dumps(r), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=4000)
    ap.add_argument("--warmup", type=int, default=50)
    ap.add_argument("--impl", default="damp", choices=["damp", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--sweep", action="store_true", help="K_hi sweep (GDN and KDA, B=256) instead of the bench line")
    ap.add_argument("--prefill", action="store_true", help="prefill chunks (64 tokens, B=256) instead of the bench line")
    ap.add_argument("--chunk-tokens", type=int, default=64, help="tokens per slot of a --prefill chunk")
    ap.add_argument("--lo-format", type=int, default=0, help="low-tier format of the --prefill workloads (0-5)")
    ap.add_argument("--prefill-kind", choices=["kda", "gdn", "both"], default="both", help="--prefill workloads")
    ap.add_argument("--prefill-batch", type=int, default=256, help="slots of the --prefill workloads (a smaller case for ncu)")
    ap.add_argument("--multitoken", action="store_true",
                    help="fused multi-token steps (T = 1..16 tokens per launch, B=256) instead of the bench line")
    ap.add_argument("--calibrate", action="store_true", help="GPU calibration run instead of the bench line")
    ap.add_argument("--drift", action="store_true", help="30-layer free-running drift run instead of the bench line")
    ap.add_argument("--tiered", action="store_true",
                    help="decay-tiered per-head K_hi (head groups) drift and step time instead of the bench line")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if args.impl == "reference":
        reference_arm(args, rank, world)
        return
    if args.sweep:
        sweep_arm(args.steps, args.warmup)
        return
    if args.prefill:
        kinds = ("kda", "gdn") if args.prefill_kind == "both" else (args.prefill_kind,)
        prefill_arm(args.steps, args.warmup, args.chunk_tokens, args.lo_format, kinds, args.prefill_batch)
        return
    if args.multitoken:
        multitoken_arm(args.steps, args.warmup)
        return
    if args.calibrate:
        calibrate_arm(args.steps, args.warmup)
        return
    if args.drift:
        drift_arm()
        return
    if args.tiered:
        tiered_arm()
        return
    import torch
    import torch.distributed as dist
    if world > 1:
        dist.init_process_group("nccl")
    try:
        r = gpu_arm(args, rank, world)
    finally:
        if world > 1 and dist.is_initialized():
            pass
    if rank == 0:
        line = make_line(r, args.steps, args.warmup, world)
        if not args.no_cpu_baseline and world == 1:
            line["cpu_baseline"] = cpu_baseline()
            line["cpu_baseline_all_cores"] = cpu_baseline_all_cores()
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
