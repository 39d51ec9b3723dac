"""Decode benchmark: BiSCo-coded Qwen3-8B linear stack on GB300.

Workload (one "step" = one decode token through every linear layer):
  the 36 layers x 7 projections of Qwen3-8B -- q_proj/o_proj 4096x4096,
  k_proj/v_proj 1024x4096, gate_proj/up_proj 12288x4096, down_proj
  4096x12288 (N x K) -- each a distinct random layer (N(0, 0.02) weights
  with 8 outlier input columns x20, drawn on the device from a seeded
  generator), coded with d = 8, base + 1 residual stage (S = 2) and 1 %
  int8 protected columns; batch 1 bf16 N(0,1) activations.  Four library
  calls per layer: bisco_gemv_multi(q, k, v), bisco_gemv(o),
  bisco_gemv_multi(gate, up), bisco_gemv(down).  The 252 coded layers hold
  5.28 GB, far more than the 129 MB L2, so every step streams its weights
  from HBM (no L2 flush needed).

Metric: decode GEMV GB/s on compressed bytes (signs + norms + int8 payload +
scales + indices) and tokens/s; value = whole-job GB/s over all ranks.

  python bench.py [--gpus N --steps K --warmup W --batch B --impl {bisco,reference}]
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "decode GEMV GB/s (compressed bytes) & tokens/s, % of HBM/tensor roofline"
ATTN = ("q_proj", "k_proj", "v_proj", "o_proj")
STACK = ("q_proj", "k_proj", "v_proj", "o_proj", "gate_proj", "up_proj", "down_proj")
# the four library calls of one layer: name, projections (indices into
# STACK) that read the same activation, and that activation's width
CALLS = (("qkv", (0, 1, 2), 4096), ("o", (3,), 4096), ("gate_up", (4, 5), 4096),
         ("down", (6,), 12288))
N_LAYERS = 36
S_STAGES = 2
RHO_PCT = 1


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--batch", type=int, default=1)
    ap.add_argument("--layers", type=int, default=N_LAYERS)
    ap.add_argument("--impl", choices=("bisco", "reference"), default="bisco")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--mode", choices=("both", "decode", "prefill", "shapes", "dense", "lora",
                                       "stack", "variants", "dominant"),
                    default="both",
                    help="decode: the GEMV step only; prefill: the tcgen05 GEMM only; "
                         "shapes: batch-1 GEMV per Qwen3-8B layer shape; lora: the decode step "
                         "with a low-rank compensation on every projection; stack: the full "
                         "7-projection stack at batch 1/4/16 and the GEMV/GEMM crossover; "
                         "variants: the decode step per protected-set / decoder variant")
    ap.add_argument("--lora-rank", type=int, default=16)
    ap.add_argument("--shape-mb", type=float, default=500.0,
                    help="--mode shapes: MB of distinct coded layers per shape (> L2)")
    ap.add_argument("--prefill-tokens", type=int, default=2048)
    ap.add_argument("--prefill-proj", default=",".join(ATTN),
                    help="--mode prefill: comma-separated Qwen3-8B projections, one layer of each")
    return ap.parse_args()


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def tensor_peaks():
    """bf16 dense tensor peaks (TFLOP/s): burst and sustained; the fp16
    kind::f16 MMA runs at the bf16 rate."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["bf16_tflops"]), float(d["bf16_tflops_sustained"]), "measured"
    except Exception:
        return 1900.0, 1700.0, "fallback"


# DRAM bytes (read + write) of one launch of the dominant call (bisco_gemv_multi
# over gate_proj + up_proj of one layer, batch 1), from the ncu capture
# summarised in profiles/ (the file gives the command), valid while the
# kernel source hashes to the recorded digest.
DOMINANT_TRAFFIC = {"bytes": 77273856, "gemv_b1_cu_sha256": "6dbd3e37908d958e777f45292efae98c6e49528de367e0741b664014b6424d48",
                    "profile": "profiles/k_gemv_b1_gate_up_b1.md"}


def dominant_traffic(B, call):
    """DRAM bytes of one dominant launch from the committed ncu capture, or
    None when the capture does not describe the kernel being timed."""
    import hashlib
    if DOMINANT_TRAFFIC["bytes"] is None or B != 1 or call != "gate_up":
        return None
    with open(os.path.join(ROOT, "paper_2607_08643_gb300", "csrc", "gemv_b1.cu"), "rb") as f:
        digest = hashlib.sha256(f.read()).hexdigest()
    return DOMINANT_TRAFFIC["bytes"] if digest == DOMINANT_TRAFFIC["gemv_b1_cu_sha256"] else None


def call_label(call, B):
    """The kernel one call of the step launches."""
    names = {"qkv": "bisco_gemv_multi q+k+v 6144x4096", "o": "bisco_gemv o_proj 4096x4096",
             "gate_up": "bisco_gemv_multi gate+up 24576x4096", "down": "bisco_gemv down_proj 4096x12288"}
    if B == 1:
        return "k_gemv_b1 (%s, batch 1, row-split table decode)" % names[call]
    return "%s, batch %d (k_gemv_stream / k_gemv MMA decode)" % (names[call], B)


def workload_config(args):
    return {
        "workload": "Qwen3-8B linear stack: %d layers x 7 projections (q/k/v/o/gate/up/down), "
                    "decode batch %d" % (args.layers, args.batch),
        "shapes_NxK": {n: list(SHAPES[n]) for n in STACK},
        "calls_per_layer": "bisco_gemv_multi(q,k,v), bisco_gemv(o), bisco_gemv_multi(gate,up), "
                           "bisco_gemv(down)",
        "chunk_dim": 8, "stages": S_STAGES, "protected_pct": RHO_PCT, "batch": args.batch,
        "weights": "N(0,0.02) + 8 outlier cols x20, seeded on device",
        "l2": "inputs larger than L2 (distinct coded layers per step, no flush)",
    }


SHAPES = {"q_proj": (4096, 4096), "k_proj": (1024, 4096), "v_proj": (1024, 4096),
          "o_proj": (4096, 4096), "gate_proj": (12288, 4096), "up_proj": (12288, 4096),
          "down_proj": (4096, 12288)}


# ---------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi clock/throttle samples taken during the timed region."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.Q,
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if not self.proc:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        mhz, mx, reasons = [], None, set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                mhz.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for nm, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        if not mhz:
            return None
        return {"sm_mhz": statistics.median(mhz), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(mhz)}


# ---------------------------------------------------------------- layers

def build_layers(args, dev):
    import torch
    from paper_2607_08643_gb300 import bisco, synth
    layers = []
    ws = None
    for l in range(args.layers):
        for j, name in enumerate(ATTN):
            N, K = synth.QWEN3_8B_SHAPES[name]
            p = synth.protected_count(K, RHO_PCT)
            W = synth.layer_weights_torch(N, K, seed=1000 * l + j, device=dev)
            need = bisco.bisco_encode_workspace_bytes(N, K)
            if ws is None or ws.numel() < need:
                ws = torch.empty(need, dtype=torch.uint8, device=dev)
            layers.append((name, bisco.bisco_encode(W, S_STAGES, p, workspace=ws)))
            del W
    torch.cuda.synchronize()
    if bisco.bisco_get_device_error() != bisco.OK:
        raise RuntimeError("device error while encoding")
    return layers


def max_over_ranks(values, world, device=None):
    """Each value's maximum over the ranks, on every rank: the job ends when
    its slowest replica does."""
    if world <= 1:
        return [float(v) for v in values]
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(v) for v in t.cpu()]


def replica_rates(world, bytes_per_step, batch, steps, ms_total, ms_e2e):
    """Whole-job rates of `world` independent replicas, each of which ran
    `steps` steps of `bytes_per_step` compressed bytes and `batch` tokens, from
    the max-over-ranks device time and end-to-end time (ms)."""
    ms_step = ms_total / steps
    return {"ms_per_step": ms_step,
            "gbs": world * bytes_per_step / (ms_step * 1e-3) / 1e9,
            "tokens_per_s": world * batch / (ms_step * 1e-3),
            "e2e_gbs": world * bytes_per_step / (ms_e2e / steps * 1e-3) / 1e9}


def build_stack(nl, dev):
    """nl layers x the 7 projections, coded with S_STAGES and RHO_PCT; list
    of per-layer lists in STACK order."""
    import torch
    from paper_2607_08643_gb300 import bisco, synth
    out, ws = [], None
    for l in range(nl):
        row = []
        for j, name in enumerate(STACK):
            N, K = SHAPES[name]
            W = synth.layer_weights_torch(N, K, seed=1000 * l + j, device=dev)
            need = bisco.bisco_encode_workspace_bytes(N, K)
            if ws is None or ws.numel() < need:
                ws = torch.empty(need, dtype=torch.uint8, device=dev)
            row.append(bisco.bisco_encode(W, S_STAGES, synth.protected_count(K, RHO_PCT), workspace=ws))
            del W
        out.append(row)
    torch.cuda.synchronize()
    if bisco.bisco_get_device_error() != bisco.OK:
        raise RuntimeError("device error while encoding the stack")
    return out


class StackIO:
    """One flat bf16 input buffer and one flat fp32 output buffer for a batch-B
    step: per layer the activations of its four calls and the outputs of its
    seven projections, with views for the calls."""

    def __init__(self, stack, B, dev, seed):
        import torch
        nl = len(stack)
        per_x = sum(k for _, _, k in CALLS) * B
        per_y = sum(SHAPES[n][0] for n in STACK) * B
        self.x = torch.empty(nl * per_x, dtype=torch.int16, device=dev)
        gen = torch.Generator(device=dev)
        gen.manual_seed(seed)
        self.x.copy_(torch.randn(self.x.numel(), generator=gen, device=dev).to(torch.bfloat16).view(torch.int16))
        self.y = torch.empty(nl * per_y, dtype=torch.float32, device=dev)
        self.xv, self.yv = [], []
        for l in range(nl):
            xo, yo, xs, ys = l * per_x, l * per_y, {}, []
            for name, _, k in CALLS:
                xs[name] = self.x[xo:xo + k * B].view(B, k)
                xo += k * B
            for n in STACK:
                N = SHAPES[n][0]
                ys.append(self.y[yo:yo + N * B].view(B, N))
                yo += N * B
            self.xv.append(xs)
            self.yv.append(ys)


def stack_step(bisco, stack, io, stream, only=None):
    """The library calls of one step (or only those of one call type)."""
    for l, row in enumerate(stack):
        for name, idx, _ in CALLS:
            if only is not None and name != only:
                continue
            x, ys = io.xv[l][name], [io.yv[l][i] for i in idx]
            if len(idx) == 1:
                bisco.bisco_gemv(row[idx[0]], x, y=ys[0], stream=stream)
            else:
                bisco.bisco_gemv_multi([row[i] for i in idx], x, ys=ys, stream=stream)


def graph_of(torch, stream, fn):
    with torch.cuda.stream(stream):
        fn()
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            fn()
    torch.cuda.synchronize()
    return g


def time_graph(torch, stream, g, steps, warmup):
    """ms per replay: CUDA events on the launching stream over `steps`
    back-to-back replays, after `warmup` untimed ones."""
    for _ in range(max(warmup, 3)):
        g.replay()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e0.record(stream)
        for _ in range(steps):
            g.replay()
        e1.record(stream)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / steps


def run_bisco(args, rank, world, local_rank):
    """The full-stack decode step (see the module docstring): timed line,
    end-to-end line, per-call rates and the dominant call's roofline."""
    import torch
    import torch.distributed as dist
    from paper_2607_08643_gb300 import bisco

    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    bisco.load()
    stack = build_stack(args.layers, dev)
    B = args.batch
    io = StackIO(stack, B, dev, seed=7 + rank)
    bytes_step = sum(L.compressed_bytes for row in stack for L in row)
    stream = torch.cuda.Stream(device=dev)
    g = graph_of(torch, stream, lambda: stack_step(bisco, stack, io, stream))
    if bisco.bisco_get_device_error(stream) != bisco.OK:
        raise RuntimeError("device error in warm-up")

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()

    for _ in range(max(args.warmup, 3)):
        g.replay()
    barrier()
    clocks = ClockSampler(local_rank)
    clocks.start()
    time.sleep(0.3)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e0.record(stream)
        for _ in range(args.steps):
            g.replay()
        e1.record(stream)
    barrier()
    ms_total = e0.elapsed_time(e1)
    clk = clocks.stop()
    if bisco.bisco_get_device_error(stream) != bisco.OK:
        raise RuntimeError("device error in timed region")

    # end to end: pinned host inputs in, graph of public-API calls, outputs out
    x_host = torch.empty(io.x.shape, dtype=torch.int16, pin_memory=True)
    x_host.copy_(io.x.cpu())
    y_host = torch.empty(io.y.shape, dtype=torch.float32, pin_memory=True)
    for _ in range(2):
        with torch.cuda.stream(stream):
            io.x.copy_(x_host, non_blocking=True)
            g.replay()
            y_host.copy_(io.y, non_blocking=True)
    barrier()
    t0 = time.perf_counter()
    f0 = torch.cuda.Event(enable_timing=True)
    f1 = torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        f0.record(stream)
        for _ in range(args.steps):
            io.x.copy_(x_host, non_blocking=True)
            g.replay()
            y_host.copy_(io.y, non_blocking=True)
        f1.record(stream)
    stream.synchronize()
    wall_e2e = time.perf_counter() - t0
    barrier()
    ms_e2e = max(f0.elapsed_time(f1), wall_e2e * 1e3)
    ms_total, ms_e2e = max_over_ranks([ms_total, ms_e2e], world, device=dev)

    # each call type alone (a graph of its launches over all layers): the
    # dominant one is the roofline line
    per_call = {}
    for name, idx, _ in CALLS:
        gc = graph_of(torch, stream, lambda n=name: stack_step(bisco, stack, io, stream, only=n))
        ms = time_graph(torch, stream, gc, args.steps, args.warmup)
        nbytes = sum(stack[0][i].compressed_bytes for i in idx)
        us = ms * 1e3 / len(stack)
        per_call[name] = {"kernel": call_label(name, B), "bytes_per_launch": nbytes,
                          "us_per_launch": us, "gbs": nbytes / (us * 1e-6) / 1e9,
                          "launches_timed": args.steps * len(stack)}
        del gc
    if bisco.bisco_get_device_error(stream) != bisco.OK:
        raise RuntimeError("device error in the per-call timing")
    dom = max(per_call, key=lambda n: per_call[n]["us_per_launch"])
    peak, peak_kind = peaks()
    for v in per_call.values():
        v["frac_of_hbm"] = v["gbs"] / peak
    d = per_call[dom]
    rates = replica_rates(world, bytes_step, B, args.steps, ms_total, ms_e2e)
    return dict(
        value=rates["gbs"], ms_per_step=rates["ms_per_step"], tokens_per_s=rates["tokens_per_s"],
        bytes_per_step=bytes_step, launches=len(CALLS) * len(stack), e2e_gbs=rates["e2e_gbs"],
        h2d=io.x.numel() * 2, d2h=io.y.numel() * 4,
        roofline={"bound": "hbm", "achieved": d["gbs"], "peak": peak, "unit": "GB/s",
                  "frac": d["gbs"] / peak, "traffic": dominant_traffic(B, dom),
                  "peak_source": "%s hbm_gbs (MEASURED_PEAKS.json, copy burst)" % peak_kind
                  if peak_kind == "measured" else "fallback 6.8 TB/s",
                  "kernel": d["kernel"], "bytes_per_launch": d["bytes_per_launch"],
                  "us_per_launch": d["us_per_launch"], "launches_timed": d["launches_timed"],
                  "step_frac_of_hbm": rates["gbs"] / world / peak},
        per_call=per_call, clocks=clk, ms_e2e=ms_e2e / args.steps, stack=stack, io=io,
        stream=stream)


def run_sweeps(args, stack, stream, dev):
    """Sub-records on the same coded stack: the decode step at batch 4 and 16
    (GEMV), and the GEMV/GEMM crossover (bisco_gemm on every projection at
    M = 1, 4, 16, 64 through the decode kernels and 128 on the tensor
    cores)."""
    import torch
    from paper_2607_08643_gb300 import bisco
    peak, _ = peaks()
    total = sum(L.compressed_bytes for row in stack for L in row)
    steps, warm = max(3, min(args.steps, 10)), 3
    sweep = []
    for B in (4, 16):
        io = StackIO(stack, B, dev, seed=100 + B)
        g = graph_of(torch, stream, lambda: stack_step(bisco, stack, io, stream))
        ms = time_graph(torch, stream, g, steps, warm)
        gbs = total / (ms * 1e-3) / 1e9
        sweep.append({"batch": B, "ms_per_step": ms, "gbs": gbs, "frac_of_hbm": gbs / peak,
                      "tokens_per_s": B / (ms * 1e-3)})
        del g, io
    cross = []
    for M in (1, 4, 16, 64, 128):
        io = StackIO(stack, M, dev, seed=200 + M)
        need = max(bisco.bisco_gemm_workspace_bytes(L, M) for row in stack for L in row)
        ws = torch.empty(max(need, 16), dtype=torch.uint8, device=dev)

        def step():
            for l, row in enumerate(stack):
                for name, idx, _ in CALLS:
                    for i in idx:
                        bisco.bisco_gemm(row[i], io.xv[l][name], Y=io.yv[l][i], workspace=ws,
                                         stream=stream)
        g = graph_of(torch, stream, step)
        ms = time_graph(torch, stream, g, steps, warm)
        cross.append({"tokens": M, "ms_per_step": ms, "tokens_per_s": M / (ms * 1e-3),
                      "gbs": total / (ms * 1e-3) / 1e9,
                      "path": "tcgen05 GEMM" if M > 16 else "decode kernels"})
        del g, io, ws
    if bisco.bisco_get_device_error(stream) != bisco.OK:
        raise RuntimeError("device error in the sweeps")
    torch.cuda.empty_cache()
    return {"decode_batch_sweep": sweep, "gemv_gemm_crossover": cross}


def run_dense_stack(args, stack, stream, dev):
    """The paper's own inference path on the same stack: every coded layer
    decoded once to dense bf16 (bisco_decode_dense), then the step as one
    cuBLAS product (torch.matmul) per call of the fused step (q/k/v and
    gate/up concatenated), at batch 1 and 16."""
    import torch
    from paper_2607_08643_gb300 import bisco
    dense = []
    for row in stack:
        mats = []
        for _, idx, k in CALLS:
            W = torch.empty((sum(row[i].N for i in idx), k), dtype=torch.bfloat16, device=dev)
            mats.append((idx, W))
        dense.append(mats)

    def materialise():
        for row, mats in zip(stack, dense):
            for idx, W in mats:
                r0 = 0
                for i in idx:
                    bisco.bisco_decode_dense(row[i], "bf16", out=W[r0:r0 + row[i].N], stream=stream)
                    r0 += row[i].N

    with torch.cuda.stream(stream):
        materialise()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e0.record(stream)
        materialise()
        e1.record(stream)
    torch.cuda.synchronize()
    if bisco.bisco_get_device_error(stream) != bisco.OK:
        raise RuntimeError("device error in bisco_decode_dense")
    ms_mat = e0.elapsed_time(e1)
    dense_bytes = sum(W.numel() * 2 for mats in dense for _, W in mats)
    out = {"how": "bisco_decode_dense to bf16 once, then torch.matmul (cuBLAS) per call: q/k/v and "
                  "gate/up concatenated, o and down alone, CUDA graph of the step",
           "materialise_ms": ms_mat, "dense_bytes_per_step": dense_bytes}
    steps = max(3, min(args.steps, 10))
    for B in (1, 16):
        xs = [[torch.randn((k, B), device=dev).to(torch.bfloat16) for _, _, k in CALLS] for _ in stack]
        ys = [[torch.empty((W.shape[0], B), dtype=torch.bfloat16, device=dev) for _, W in mats] for mats in dense]

        def step():
            for l, mats in enumerate(dense):
                for c, (_, W) in enumerate(mats):
                    torch.matmul(W, xs[l][c], out=ys[l][c])
        g = graph_of(torch, stream, step)
        ms = time_graph(torch, stream, g, steps, 3)
        out["batch_%d" % B] = {"ms_per_step": ms, "tokens_per_s": B / (ms * 1e-3),
                               "dense_gbs": dense_bytes / (ms * 1e-3) / 1e9}
        del g, xs, ys
    del dense
    torch.cuda.empty_cache()
    return out


def run_residual_decode(args, stack, stream, dev):
    """Load-time decode of the whole stack to fp32 (Sec. III-G): packed (all
    stages in one pass, bisco_decode_dense) against sequential (one pass per
    stage, bisco_decode_dense_stage accumulating into the output).  Every
    layer is decoded into one reused fp32 buffer of its shape."""
    import torch
    from paper_2607_08643_gb300 import bisco
    bufs = {SHAPES[n]: torch.empty(SHAPES[n], dtype=torch.float32, device=dev) for n in STACK}

    def packed():
        for row in stack:
            for L in row:
                bisco.bisco_decode_dense(L, "f32", out=bufs[(L.N, L.K)], stream=stream)

    def sequential():
        for row in stack:
            for L in row:
                bisco.bisco_decode_dense_sequential(L, out=bufs[(L.N, L.K)], stream=stream)

    out = {}
    for name, fn in (("packed", packed), ("sequential", sequential)):
        g = graph_of(torch, stream, fn)
        out[name + "_ms"] = time_graph(torch, stream, g, 3, 2)
        del g
    if bisco.bisco_get_device_error(stream) != bisco.OK:
        raise RuntimeError("device error in the residual decode")
    elems = sum(L.N * L.K for row in stack for L in row)
    coded = sum(L.compressed_bytes for row in stack for L in row)
    out.update({"layers": len(stack) * len(STACK), "stages": S_STAGES, "dense_fp32_bytes": 4 * elems,
                "compressed_bytes": coded,
                "packed_gbs": (coded + 4 * elems) / (out["packed_ms"] * 1e-3) / 1e9,
                "sequential_over_packed": out["sequential_ms"] / out["packed_ms"],
                "how": "CUDA graph of one decode of every layer of the stack into a reused fp32 "
                       "buffer per shape; sequential = S passes (write, then read-add-write)"})
    del bufs
    torch.cuda.empty_cache()
    return out


def run_prefill_stack(args, stack, stream, dev):
    """Prefill on the tensor cores: bisco_gemm on the 7 projections of the
    first 4 layers of the stack at --prefill-tokens tokens, a CUDA graph of
    the 28 calls; TFLOP/s on the algorithmic 2*M*N*K."""
    import torch
    from paper_2607_08643_gb300 import bisco
    M = args.prefill_tokens
    rows = stack[:4]
    X = {k: torch.randn((M, k), device=dev).to(torch.bfloat16).view(torch.int16) for k in (4096, 12288)}
    Ys = [[torch.empty((M, L.N), device=dev) for L in row] for row in rows]
    ws = torch.empty(max(bisco.bisco_gemm_workspace_bytes(L, M) for row in rows for L in row),
                     dtype=torch.uint8, device=dev)

    def step():
        for row, ys in zip(rows, Ys):
            for L, Y in zip(row, ys):
                bisco.bisco_gemm(L, X[L.K], Y=Y, workspace=ws, stream=stream)
    g = graph_of(torch, stream, step)
    ms = time_graph(torch, stream, g, max(3, min(args.steps, 10)), 3)
    if bisco.bisco_get_device_error(stream) != bisco.OK:
        raise RuntimeError("device error in prefill")
    flops = sum(2.0 * M * L.N * L.K for row in rows for L in row)
    tf = flops / (ms * 1e-3) / 1e12
    # each projection alone: a graph of its 4 calls
    per_proj = {}
    for j, name in enumerate(STACK):
        def one(j=j):
            for row, ys in zip(rows, Ys):
                bisco.bisco_gemm(row[j], X[row[j].K], Y=ys[j], workspace=ws, stream=stream)
        gj = graph_of(torch, stream, one)
        msj = time_graph(torch, stream, gj, max(3, min(args.steps, 10)), 3)
        fj = sum(2.0 * M * row[j].N * row[j].K for row in rows)
        per_proj[name] = {"us_per_call": round(msj * 1e3 / len(rows), 2),
                          "tflops": round(fj / (msj * 1e-3) / 1e12, 1)}
        del gj
    if bisco.bisco_get_device_error(stream) != bisco.OK:
        raise RuntimeError("device error in prefill")
    burst, sustained, kind = tensor_peaks()
    del g, X, Ys, ws
    torch.cuda.empty_cache()
    return {"metric": "prefill GEMM TFLOP/s (2*M*N*K, decoded weight never written)",
            "workload": "Qwen3-8B 7 projections x 4 layers, %d tokens, S=%d, %d%% protected"
                        % (M, S_STAGES, RHO_PCT),
            "value": tf, "unit": "TFLOP/s", "ms_per_step": ms,
            "roofline": {"bound": "tensor", "achieved": tf, "peak": burst, "unit": "TFLOP/s",
                         "frac": tf / burst, "frac_of_sustained": tf / sustained,
                         "peak_source": "%s bf16_tflops (MEASURED_PEAKS.json; fp16 rate = bf16)" % kind,
                         "kernels": "k_gemm_prep + k_gemm per projection, + k_gemm_fixup where "
                                    "the call splits tiles (stream-K)"},
            "per_projection": per_proj,
            "dtype": "f16 x f16 -> f32"}


# ---------------------------------------------------------------- prefill

def run_prefill(args, local_rank):
    """Prefill (bisco_gemm on the tensor cores): one layer of each projection
    in --prefill-proj (default the four attention projections) at M tokens, a
    CUDA graph of the calls (fp16 pre-pass + tcgen05 kernel each, plus the
    fixup kernel where a call splits tiles), CUDA events over `steps`
    replays.  TFLOP/s on the algorithmic 2*M*N*K."""
    import torch
    from paper_2607_08643_gb300 import bisco, synth
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    M = args.prefill_tokens
    names = [n for n in args.prefill_proj.split(",") if n]
    if not names or any(n not in synth.QWEN3_8B_SHAPES for n in names):
        raise SystemExit("--prefill-proj: names from %s" % ",".join(synth.QWEN3_8B_SHAPES))
    layers = []
    for j, name in enumerate(names):
        N, K = synth.QWEN3_8B_SHAPES[name]
        W = synth.layer_weights_torch(N, K, seed=500 + j, device=dev)
        layers.append((name, bisco.bisco_encode(W, S_STAGES, synth.protected_count(K, RHO_PCT))))
        del W
    Xk = {K: torch.randn((M, K), device=dev).to(torch.bfloat16).view(torch.int16)
          for K in sorted({L.K for _, L in layers})}
    Ys = [torch.empty((M, L.N), device=dev) for _, L in layers]
    ws = torch.empty(max(bisco.bisco_gemm_workspace_bytes(L, M) for _, L in layers),
                     dtype=torch.uint8, device=dev)
    torch.cuda.synchronize()
    stream = torch.cuda.Stream(device=dev)
    with torch.cuda.stream(stream):
        for (_, L), Y in zip(layers, Ys):
            bisco.bisco_gemm(L, Xk[L.K], Y=Y, workspace=ws, stream=stream)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for (_, L), Y in zip(layers, Ys):
                bisco.bisco_gemm(L, Xk[L.K], Y=Y, workspace=ws, stream=stream)
    torch.cuda.synchronize()
    for _ in range(max(args.warmup, 3)):
        g.replay()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e0.record(stream)
        for _ in range(args.steps):
            g.replay()
        e1.record(stream)
    torch.cuda.synchronize()
    if bisco.bisco_get_device_error(stream) != bisco.OK:
        raise RuntimeError("device error in prefill")
    ms = e0.elapsed_time(e1) / args.steps
    flops = sum(2.0 * M * L.N * L.K for _, L in layers)
    tf = flops / (ms * 1e-3) / 1e12
    burst, sustained, kind = tensor_peaks()
    return {"metric": "prefill GEMM TFLOP/s (2*M*N*K, decoded weight never written)",
            "workload": "Qwen3-8B %s, one layer each, %d tokens, S=%d, %d%% protected"
                        % ("/".join(names), M, S_STAGES, RHO_PCT),
            "value": tf, "unit": "TFLOP/s", "ms_per_step": ms, "tokens_per_s": M / (ms * 1e-3),
            "roofline": {"bound": "tensor", "achieved": tf, "peak": burst, "unit": "TFLOP/s",
                         "frac": tf / burst, "frac_of_sustained": tf / sustained,
                         "peak_source": "%s bf16_tflops (MEASURED_PEAKS.json; fp16 rate = bf16)" % kind,
                         "kernels": "k_gemm_prep + k_gemm per projection, + k_gemm_fixup where "
                                    "the call splits tiles (stream-K)"},
            "dtype": "f16 x f16 -> f32"}


# ------------------------------------------------------------------ dense

def run_dense(args, local_rank):
    """The materialise-then-multiply comparison: the same 36-layer q/k/v/o
    stack decoded once to dense bf16 weights with bisco_decode_dense (q/k/v
    of a layer into one [6144][4096] matrix), then the decode step as two
    cuBLAS products per layer (torch.matmul, a CUDA graph of the step), the
    same launch structure as the fused step.  Reports the one-time decode
    and the dense step (its GB/s counts the dense bf16 weight bytes)."""
    import torch
    from paper_2607_08643_gb300 import bisco
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    bisco.load()
    layers = build_layers(args, dev)
    B, K = args.batch, 4096
    dense = []
    for li in range(args.layers):
        qkv = [layers[4 * li + j][1] for j in range(3)]
        W_qkv = torch.empty((sum(L.N for L in qkv), K), dtype=torch.bfloat16, device=dev)
        W_o = torch.empty((layers[4 * li + 3][1].N, K), dtype=torch.bfloat16, device=dev)
        dense.append((qkv, W_qkv, layers[4 * li + 3][1], W_o))
    stream = torch.cuda.Stream(device=dev)

    def materialise():
        for qkv, W_qkv, L_o, W_o in dense:
            r0 = 0
            for L in qkv:
                bisco.bisco_decode_dense(L, "bf16", out=W_qkv[r0:r0 + L.N], stream=stream)
                r0 += L.N
            bisco.bisco_decode_dense(L_o, "bf16", out=W_o, stream=stream)

    with torch.cuda.stream(stream):
        materialise()   # warm-up
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e0.record(stream)
        materialise()
        e1.record(stream)
    torch.cuda.synchronize()
    if bisco.bisco_get_device_error(stream) != bisco.OK:
        raise RuntimeError("device error in bisco_decode_dense")
    ms_mat = e0.elapsed_time(e1)
    comp = sum(L.compressed_bytes for _, L in layers)
    dense_bytes = sum((W_qkv.numel() + W_o.numel()) * 2 for _, W_qkv, _, W_o in dense)

    x = torch.randn((2 * args.layers, K, B), device=dev).to(torch.bfloat16)
    ys = [(torch.empty((W_qkv.shape[0], B), dtype=torch.bfloat16, device=dev),
           torch.empty((W_o.shape[0], B), dtype=torch.bfloat16, device=dev)) for _, W_qkv, _, W_o in dense]

    def step():
        for li, (_, W_qkv, _, W_o) in enumerate(dense):
            torch.matmul(W_qkv, x[2 * li], out=ys[li][0])
            torch.matmul(W_o, x[2 * li + 1], out=ys[li][1])

    with torch.cuda.stream(stream):
        step()
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            step()
    torch.cuda.synchronize()
    for _ in range(max(args.warmup, 3)):
        g.replay()
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        e0.record(stream)
        for _ in range(args.steps):
            g.replay()
        e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / args.steps
    return {"how": "bisco_decode_dense to bf16 once, then torch.matmul (cuBLAS) per step: "
                   "q/k/v concatenated + o_proj per layer, CUDA graph",
            "materialise_ms": ms_mat,
            "materialise_gbs": (comp + dense_bytes) / (ms_mat * 1e-3) / 1e9,
            "dense_bytes_per_step": dense_bytes, "compressed_bytes": comp,
            "ms_per_step": ms, "tokens_per_s": B / (ms * 1e-3),
            "dense_gbs": dense_bytes / (ms * 1e-3) / 1e9, "batch": B}


# ------------------------------------------------------------------- lora

def run_lora(args, local_rank):
    """Low-rank compensation (rank --lora-rank) on every projection of the
    36-layer q/k/v/o decode step.  Times the step without it, with it fused
    into the GEMV at batch 1 (bisco_gemv_multi_lora for q/k/v,
    bisco_gemv_lora for o: one launch each, as without it), and with the
    two-kernel bisco_lora_apply after each GEMV (CUDA graphs of the same
    calls, CUDA events over `steps` replays); and that two-kernel
    compensation alone: a graph of its calls for every projection, timed
    replay by replay with L2 flushed in between (the adapters of the stack
    are smaller than L2).  Adapter bytes are rank * (K + N) bf16 per
    projection; the roofline counts those plus x, t and the read-modify-
    write of y."""
    import torch
    from paper_2607_08643_gb300 import bisco
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    bisco.load()
    layers = build_layers(args, dev)
    B, K, R = args.batch, 4096, args.lora_rank
    gen = torch.Generator(device=dev)
    gen.manual_seed(4242)
    adapters = []
    for _, L in layers:
        A = (torch.randn((R, L.K), generator=gen, device=dev) / L.K ** 0.5).to(torch.bfloat16)
        Bm = (torch.randn((L.N, R), generator=gen, device=dev) * 0.02).to(torch.bfloat16)
        adapters.append((A, Bm))
    x = torch.randn((2 * args.layers, B, K), generator=gen, device=dev).to(torch.bfloat16)
    ys = [torch.zeros((B, L.N), dtype=torch.float32, device=dev) for _, L in layers]
    t = torch.empty((B, R), dtype=torch.float32, device=dev)
    stream = torch.cuda.Stream(device=dev)

    fused_ok = B == 1

    def step(with_lora, with_gemv=True, fused=False):
        if fused:
            for li in range(args.layers):
                q = [4 * li + j for j in range(3)]
                bisco.bisco_gemv_multi_lora([layers[i][1] for i in q],
                                            [adapters[i] + (1.0,) for i in q], x[2 * li],
                                            ys=[ys[i] for i in q], stream=stream)
                o = 4 * li + 3
                bisco.bisco_gemv_lora(layers[o][1], adapters[o] + (1.0,), x[2 * li + 1], y=ys[o],
                                      stream=stream)
            return
        for li in range(args.layers):
            q = [4 * li + j for j in range(3)]
            if with_gemv:
                bisco.bisco_gemv_multi([layers[i][1] for i in q], x[2 * li],
                                       ys=[ys[i] for i in q], stream=stream)
            if with_lora:
                for i in q:
                    bisco.bisco_lora_apply(*adapters[i], x[2 * li], ys[i], 1.0, t=t, stream=stream)
            o = 4 * li + 3
            if with_gemv:
                bisco.bisco_gemv(layers[o][1], x[2 * li + 1], y=ys[o], stream=stream)
            if with_lora:
                bisco.bisco_lora_apply(*adapters[o], x[2 * li + 1], ys[o], 1.0, t=t, stream=stream)

    graphs = {}
    variants = {"plain": (False, True, False), "lora": (True, True, False), "only": (True, False, False)}
    if fused_ok:
        variants["fused"] = (True, True, True)
    for key, (wl, wg, fu) in variants.items():
        with torch.cuda.stream(stream):
            step(wl, wg, fu)
            torch.cuda.synchronize()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                step(wl, wg, fu)
        graphs[key] = g
    torch.cuda.synchronize()
    if bisco.bisco_get_device_error(stream) != bisco.OK:
        raise RuntimeError("device error in the lora step")
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ms = {}
    for key in [k for k in ("plain", "lora", "fused") if k in graphs]:
        for _ in range(max(args.warmup, 3)):
            graphs[key].replay()
        torch.cuda.synchronize()
        with torch.cuda.stream(stream):
            e0.record(stream)
            for _ in range(args.steps):
                graphs[key].replay()
            e1.record(stream)
        torch.cuda.synchronize()
        ms[key] = e0.elapsed_time(e1) / args.steps
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    only = []
    for it in range(max(args.warmup, 3) + args.steps):
        with torch.cuda.stream(stream):
            flush.fill_(it & 255)
            e0.record(stream)
            graphs["only"].replay()
            e1.record(stream)
        torch.cuda.synchronize()
        if it >= max(args.warmup, 3):
            only.append(e0.elapsed_time(e1))
    ms_only = sum(only) / len(only)
    calls = len(layers)
    adapter_bytes = sum((A.numel() + Bm.numel()) * 2 for A, Bm in adapters)
    io_bytes = sum(B * (L.K * 2 + L.N * 8) + 2 * B * R * 4 for _, L in layers)
    peak, peak_kind = peaks()
    gbs = (adapter_bytes + io_bytes) / (ms_only * 1e-3) / 1e9
    return {"metric": "decode step with low-rank compensation on every projection",
            "rank": R, "batch": B, "layers": args.layers,
            "step_ms_without": ms["plain"],
            "fused": ({"step_ms": ms["fused"], "overhead_pct": 100.0 * (ms["fused"] / ms["plain"] - 1.0),
                       "tokens_per_s": B / (ms["fused"] * 1e-3),
                       "kernels": "k_gemv_b1 with t = A x and Bm t in the same launch"}
                      if "fused" in ms else None),
            "step_ms_with": ms["lora"],
            "overhead_pct": 100.0 * (ms["lora"] / ms["plain"] - 1.0),
            "tokens_per_s_with": B / (ms["lora"] * 1e-3),
            "compensation_alone": {"ms_per_step": ms_only, "calls": calls,
                                   "us_per_call": ms_only * 1e3 / calls,
                                   "adapter_bytes": adapter_bytes, "io_bytes": io_bytes,
                                   "gbs": gbs, "frac_of_hbm": gbs / peak,
                                   "peak_source": peak_kind,
                                   "l2": "flushed (256 MB write) before every replay"},
            "kernels": "step_ms_with: the GEMV, then k_lora_down + k_lora_up per projection"}


# ----------------------------------------------------------------- shapes

def run_shapes(args, local_rank):
    """Batch-1 bisco_gemv per Qwen3-8B linear shape: a CUDA graph of one call
    on each of about --shape-mb MB of distinct coded layers of that shape
    (larger than L2, so every call streams from HBM), CUDA events over
    `steps` replays; GB/s on the algorithmic compressed bytes.  Attention
    shapes use S=2 and 1 % protection (N(0,0.02) weights), MLP shapes S=3
    and 2 % (Student-t(4) weights), as in the paper-derived configurations."""
    import torch
    from paper_2607_08643_gb300 import bisco, synth
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    peak, _ = peaks()
    out = []
    for name, (N, K) in synth.QWEN3_8B_SHAPES.items():
        mlp = name in synth.MLP
        S, rho, dist = (3, 2, "t4") if mlp else (2, 1, "normal")
        p = synth.protected_count(K, rho)
        one = S * N * (K // 8) * 3 + N * p + 6 * p
        nl = max(4, int(args.shape_mb * 1e6 / one))
        W = synth.layer_weights_torch(N, K, seed=900, device=dev, dist=dist)
        ws = torch.empty(bisco.bisco_encode_workspace_bytes(N, K), dtype=torch.uint8, device=dev)
        layers = [bisco.bisco_encode(W, S, p, workspace=ws) for _ in range(nl)]
        del W
        xs = torch.randn((nl, 1, K), device=dev).to(torch.bfloat16).view(torch.int16)
        ys = torch.empty((nl, 1, N), device=dev)
        torch.cuda.synchronize()
        stream = torch.cuda.Stream(device=dev)
        with torch.cuda.stream(stream):
            for i, L in enumerate(layers):
                bisco.bisco_gemv(L, xs[i], y=ys[i], stream=stream)
            torch.cuda.synchronize()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                for i, L in enumerate(layers):
                    bisco.bisco_gemv(L, xs[i], y=ys[i], stream=stream)
        torch.cuda.synchronize()
        for _ in range(max(args.warmup, 3)):
            g.replay()
        torch.cuda.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            e0.record(stream)
            for _ in range(args.steps):
                g.replay()
            e1.record(stream)
        torch.cuda.synchronize()
        if bisco.bisco_get_device_error(stream) != bisco.OK:
            raise RuntimeError("device error in shape sweep")
        us = e0.elapsed_time(e1) * 1e3 / (args.steps * nl)
        gbs = one / (us * 1e-6) / 1e9
        out.append({"shape": name, "N": N, "K": K, "S": S, "p": p, "layers": nl,
                    "bytes_per_launch": one, "us_per_launch": us, "gbs": gbs,
                    "frac_of_hbm": gbs / peak})
        del layers, xs, ys, g
        torch.cuda.empty_cache()
    return out


# --------------------------------------------------------------- variants

def run_variants(args, local_rank):
    """The batch-B decode step of the 36-layer q/k/v/o stack (as in the
    default line) with each protected-set and decoder variant of the
    library: INT8 protected columns (the default), FP8 E4M3 and BF16
    payloads (protected-format ablation), 1 % protected output rows
    (Eq. 9 / Eq. 10 on rows) and the learned decoder step as per-stage
    tables (bisco_gemv_table, one call per projection).  One CUDA graph per
    variant, CUDA events over `steps` replays; GB/s on each variant's own
    compressed bytes (the decoder tables, 8 KB per layer, are not counted).
    Then the gated MLP of the same layers (gate/up grouped, down) with
    per-layer INT8 columns and with the coupled set of Eq. 9, and the
    prefill GEMM of q_proj-shaped layers per variant (its epilogue kernels
    included)."""
    import torch
    from paper_2607_08643_gb300 import bisco, synth
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    peak, peak_kind = peaks()
    B = args.batch
    gen = torch.Generator(device=dev)
    gen.manual_seed(31)
    x = torch.randn((B, 4096), generator=gen, device=dev).to(torch.bfloat16).view(torch.int16)
    stream = torch.cuda.Stream(device=dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    tabs = (torch.randn((S_STAGES, 256, 8), generator=gen, device=dev) * 0.35).to(torch.float16)
    out = []
    for name, axis, fmt, table in (("int8 columns", 0, bisco.PROT_INT8, False),
                                   ("fp8 e4m3 columns", 0, bisco.PROT_E4M3, False),
                                   ("bf16 columns", 0, bisco.PROT_BF16, False),
                                   ("int8 rows", 1, bisco.PROT_INT8, False),
                                   ("decoder tables", 0, bisco.PROT_INT8, True)):
        layers = []
        for l in range(args.layers):
            for j, proj in enumerate(ATTN):
                N, K = synth.QWEN3_8B_SHAPES[proj]
                p = synth.protected_count(N if axis else K, RHO_PCT)
                W = synth.layer_weights_torch(N, K, seed=1000 * l + j, device=dev)
                layers.append(bisco.bisco_encode(W, S_STAGES, p, axis=axis, fmt=fmt))
                del W
        ys = [torch.empty((B, L.N), device=dev) for L in layers]
        torch.cuda.synchronize()

        def step():
            for l in range(args.layers):
                q = list(range(4 * l, 4 * l + 4))
                if table:
                    for i in q:
                        bisco.bisco_gemv_table(layers[i], tabs, x, y=ys[i], stream=stream)
                else:
                    bisco.bisco_gemv_multi([layers[i] for i in q[:3]], x,
                                           ys=[ys[i] for i in q[:3]], stream=stream)
                    bisco.bisco_gemv(layers[q[3]], x, y=ys[q[3]], stream=stream)

        with torch.cuda.stream(stream):
            step()
            torch.cuda.synchronize()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                step()
        torch.cuda.synchronize()
        for _ in range(max(args.warmup, 3)):
            g.replay()
        torch.cuda.synchronize()
        with torch.cuda.stream(stream):
            e0.record(stream)
            for _ in range(args.steps):
                g.replay()
            e1.record(stream)
        torch.cuda.synchronize()
        if bisco.bisco_get_device_error(stream) != bisco.OK:
            raise RuntimeError("device error in variant " + name)
        ms = e0.elapsed_time(e1) / args.steps
        total = sum(L.compressed_bytes for L in layers)
        gbs = total / (ms * 1e-3) / 1e9
        out.append({"variant": name, "bytes_per_step": total, "ms_per_step": ms, "gbs": gbs,
                    "frac_of_hbm": gbs / peak, "tokens_per_s": B / (ms * 1e-3)})
        del layers, ys, g
        torch.cuda.empty_cache()
    # the gated MLP (gate/up 12288x4096, down 4096x12288): 1 % protected input
    # columns per layer, against the coupled set of Eq. 9 (rows of gate and
    # up, columns of down, 1 % of the 12288 channels)
    xf = torch.randn((B, 12288), generator=gen, device=dev).to(torch.bfloat16).view(torch.int16)
    mlp = []
    for name in ("int8 columns", "coupled rows + columns"):
        layers = []
        for l in range(args.layers):
            Ws = [synth.layer_weights_torch(*synth.QWEN3_8B_SHAPES[proj], seed=1000 * l + 4 + j,
                                            device=dev)
                  for j, proj in enumerate(("gate_proj", "up_proj", "down_proj"))]
            if name == "int8 columns":
                layers += [bisco.bisco_encode(W, S_STAGES, synth.protected_count(W.shape[1], RHO_PCT))
                           for W in Ws]
            else:
                idx = bisco.bisco_select_coupled(Ws[0], Ws[1], Ws[2],
                                                 synth.protected_count(Ws[0].shape[0], RHO_PCT))
                layers += [bisco.bisco_encode_with_set(Ws[0], S_STAGES, idx, axis=1),
                           bisco.bisco_encode_with_set(Ws[1], S_STAGES, idx, axis=1),
                           bisco.bisco_encode_with_set(Ws[2], S_STAGES, idx, axis=0)]
            del Ws
        ys = [torch.empty((B, L.N), device=dev) for L in layers]
        torch.cuda.synchronize()

        def step():
            for l in range(args.layers):
                g = 3 * l
                bisco.bisco_gemv_multi(layers[g:g + 2], x, ys=ys[g:g + 2], stream=stream)
                bisco.bisco_gemv(layers[g + 2], xf, y=ys[g + 2], stream=stream)

        with torch.cuda.stream(stream):
            step()
            torch.cuda.synchronize()
            gr = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gr, stream=stream):
                step()
        torch.cuda.synchronize()
        for _ in range(max(args.warmup, 3)):
            gr.replay()
        torch.cuda.synchronize()
        with torch.cuda.stream(stream):
            e0.record(stream)
            for _ in range(args.steps):
                gr.replay()
            e1.record(stream)
        torch.cuda.synchronize()
        if bisco.bisco_get_device_error(stream) != bisco.OK:
            raise RuntimeError("device error in MLP variant " + name)
        ms = e0.elapsed_time(e1) / args.steps
        total = sum(L.compressed_bytes for L in layers)
        gbs = total / (ms * 1e-3) / 1e9
        mlp.append({"variant": name, "bytes_per_step": total, "ms_per_step": ms, "gbs": gbs,
                    "frac_of_hbm": gbs / peak, "tokens_per_s": B / (ms * 1e-3)})
        del layers, ys, gr
        torch.cuda.empty_cache()
    # prefill: bisco_gemm on 8 distinct q_proj-shaped layers per variant at
    # --prefill-tokens, the variants' epilogue kernels included
    M = args.prefill_tokens
    Xp = torch.randn((M, 4096), generator=gen, device=dev).to(torch.bfloat16).view(torch.int16)
    tf_burst, _, _ = tensor_peaks()
    pre = []
    for name, axis, fmt in (("int8 columns", 0, bisco.PROT_INT8),
                            ("fp8 e4m3 columns", 0, bisco.PROT_E4M3),
                            ("int8 rows", 1, bisco.PROT_INT8)):
        layers = []
        for l in range(8):
            W = synth.layer_weights_torch(4096, 4096, seed=5000 + l, device=dev)
            layers.append(bisco.bisco_encode(W, S_STAGES, synth.protected_count(4096, RHO_PCT),
                                             axis=axis, fmt=fmt))
            del W
        need = max(bisco.bisco_gemm_workspace_bytes(L, M) for L in layers)
        gws = torch.empty(max(need, 16), dtype=torch.uint8, device=dev)
        Y = torch.empty((M, 4096), device=dev)
        torch.cuda.synchronize()

        def step():
            for L in layers:
                bisco.bisco_gemm(L, Xp, Y=Y, workspace=gws, stream=stream)

        with torch.cuda.stream(stream):
            step()
            torch.cuda.synchronize()
            gp = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gp, stream=stream):
                step()
        torch.cuda.synchronize()
        for _ in range(max(args.warmup, 3)):
            gp.replay()
        torch.cuda.synchronize()
        with torch.cuda.stream(stream):
            e0.record(stream)
            for _ in range(args.steps):
                gp.replay()
            e1.record(stream)
        torch.cuda.synchronize()
        if bisco.bisco_get_device_error(stream) != bisco.OK:
            raise RuntimeError("device error in prefill variant " + name)
        us = e0.elapsed_time(e1) * 1e3 / (args.steps * len(layers))
        tflops = 2.0 * M * 4096 * 4096 / (us * 1e-6) / 1e12
        pre.append({"variant": name, "tokens": M, "us_per_layer": us, "tflops": tflops,
                    "frac_of_tensor_burst": tflops / tf_burst})
        del layers, gws, Y, gp
        torch.cuda.empty_cache()
    return {"metric": "decode step per protected-set / decoder variant", "unit": "GB/s",
            "batch": B, "layers": args.layers, "hbm_peak_gbs": peak, "peak_source": peak_kind,
            "variants": out, "mlp_variants": mlp, "prefill_q_proj": pre}


# ------------------------------------------------------------ CPU oracle

# Rows of each projection shape a CPU worker codes and applies repeatedly: a
# bounded sample of the same workload (every byte of a coded layer costs the
# oracle the same work, so a slab of rows stands for the layer).
ORACLE_ROWS = {4096: 256, 12288: 128}
_WORKER_LAYER = {}


def _oracle_worker(task):
    """One CPU process of the oracle baseline: codes a slab of rows of one
    projection shape with the fp64 oracle (once per process), then applies it
    to a batch of activations (decode to dense + naive matmul) until
    `seconds` have passed.  Returns (compressed bytes processed, seconds,
    calls)."""
    name, seconds, batch = task
    import oracle
    from paper_2607_08643_gb300 import synth
    N, K = SHAPES[name]
    key = (name, batch)
    if key not in _WORKER_LAYER:
        rows = ORACLE_ROWS[K]
        L = oracle.encode(synth.layer_weights(rows, K, seed=STACK.index(name)), S=S_STAGES,
                          p=synth.protected_count(K, RHO_PCT))
        _WORKER_LAYER[key] = (L, synth.activations(batch, K, seed=99))
    L, X = _WORKER_LAYER[key]
    per_call = S_STAGES * L["N"] * (K // 8) * 3 + L["N"] * L["p"] + 6 * L["p"]
    n, t0 = 0, time.perf_counter()
    while True:
        oracle.gemv(L, X)
        n += 1
        el = time.perf_counter() - t0
        if el >= seconds:
            return n * per_call, el, n


class OraclePool:
    """The oracle on `workers` host processes (spawned, so that no process
    forks after CUDA work), each on one projection shape of the stack in
    turn; rate = all bytes / the slowest worker's time."""

    def __init__(self, workers):
        import multiprocessing as mp
        self.workers = workers
        self.pool = mp.get_context("spawn").Pool(workers) if workers > 1 else None

    def sample(self, seconds, batch):
        tasks = [(STACK[w % len(STACK)], seconds, batch) for w in range(self.workers)]
        res = self.pool.map(_oracle_worker, tasks) if self.pool else [_oracle_worker(tasks[0])]
        nbytes = sum(r[0] for r in res)
        el = max(r[1] for r in res)
        return nbytes / el / 1e9, el, sum(r[2] for r in res)

    def close(self):
        if self.pool:
            self.pool.close()
            self.pool.join()


def host_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def cpu_baseline(seconds, batch):
    """The fp64 oracle as it stands on the host cores, single-process and on
    every core, on a bounded sample of the stack's workload."""
    cores = host_cores()
    one = OraclePool(1)
    gbs1, el1, n1 = one.sample(seconds / 2, batch)
    allp = OraclePool(cores)
    allp.sample(0.5, batch)   # every worker codes its slab once
    gbs, el, n = allp.sample(seconds / 2, batch)
    allp.close()
    slab = ", ".join("%d rows of %s" % (ORACLE_ROWS[SHAPES[nm][1]], nm) for nm in STACK)
    return {"value": gbs, "unit": "GB/s", "cores": cores, "kind": "oracle",
            "sample": "fp64 decode-to-dense + naive matmul of coded row slabs (%s), one shape "
                      "per process, %d processes for %.1f s (%d calls), batch %d" % (slab, cores, el, n, batch),
            "single_core": {"value": gbs1, "unit": "GB/s", "cores": 1,
                            "sample": "q_proj slab, %.1f s (%d calls)" % (el1, n1)},
            "host_cores_available": cores}


def run_reference(args, rank, world):
    """Reference arm: the CPU oracle as it stands, on every host core, on the
    same metric; each step is a bounded sample of the workload (all workers
    for a fixed time), timed as a step."""
    if rank != 0:
        return None
    cores = host_cores()
    pool = OraclePool(cores)
    per_step = max(0.5, min(10.0, 120.0 / max(1, args.steps + args.warmup)))
    for _ in range(args.warmup):
        pool.sample(per_step, args.batch)
    vals, secs, t0 = [], [], time.perf_counter()
    for _ in range(args.steps):
        gbs, el, _ = pool.sample(per_step, args.batch)
        vals.append(gbs)
        secs.append(el)
    wall = time.perf_counter() - t0
    pool.close()
    gbs = statistics.median(vals)
    slab = ", ".join("%d rows of %s" % (ORACLE_ROWS[SHAPES[nm][1]], nm) for nm in STACK)
    return {
        "impl": "reference", "metric": METRIC, "value": gbs, "unit": "GB/s", "n_gpus": 1,
        "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": statistics.median(secs) * 1e3,
        "step": "a bounded sample of the workload: every host core runs the oracle on coded row "
                "slabs of one projection shape for %.1f s; value = the sample's compressed bytes "
                "/ its time" % per_step,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": workload_config(args),
        "cpu_baseline": {"kind": "oracle", "cores": cores, "value": gbs, "unit": "GB/s",
                         "sample": "fp64 decode-to-dense + naive matmul on %s; %d processes"
                                   % (slab, cores)},
        "e2e": {"value": gbs, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "wall_s": wall,
    }


def main():
    args = parse()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        import torch
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl")
    if args.impl == "reference":
        line = run_reference(args, rank, world)
        if line is not None:
            print(json.dumps(line))
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()
        return
    if args.mode == "shapes":
        res = run_shapes(args, local_rank)
        if rank == 0:
            print(json.dumps({"metric": "batch-1 GEMV GB/s per Qwen3-8B shape (compressed bytes)",
                              "unit": "GB/s", "hbm_peak_gbs": peaks()[0], "steps": args.steps,
                              "data": "synthetic", "shapes": res}))
        return
    if args.mode == "variants":
        vr = run_variants(args, local_rank)
        if rank == 0:
            print(json.dumps(dict(vr, n_gpus=world, steps=args.steps, warmup=args.warmup,
                                  data="synthetic", config=workload_config(args))))
        return
    if args.mode == "dominant":
        # the dominant call alone, launched directly (no graph), for an ncu
        # capture of one launch on a small stack: python bench.py --mode
        # dominant --layers 2 --steps 2 --warmup 1
        import torch
        from paper_2607_08643_gb300 import bisco
        dev = torch.device("cuda", local_rank)
        torch.cuda.set_device(dev)
        stack = build_stack(args.layers, dev)
        io = StackIO(stack, args.batch, dev, seed=7)
        stream = torch.cuda.Stream(device=dev)
        with torch.cuda.stream(stream):
            for _ in range(args.warmup + args.steps):
                stack_step(bisco, stack, io, stream, only="gate_up")
        torch.cuda.synchronize()
        if bisco.bisco_get_device_error(stream) != bisco.OK:
            raise RuntimeError("device error")
        print(json.dumps({"mode": "dominant", "kernel": call_label("gate_up", args.batch),
                          "launches": len(stack) * (args.warmup + args.steps),
                          "bytes_per_launch": sum(stack[0][i].compressed_bytes for i in (4, 5))}))
        return
    if args.mode == "lora":
        lr = run_lora(args, local_rank)
        if rank == 0:
            print(json.dumps(dict(lr, n_gpus=world, steps=args.steps, warmup=args.warmup,
                                  data="synthetic", config=workload_config(args))))
        return
    if args.mode == "dense":
        dn = run_dense(args, local_rank)
        if rank == 0:
            print(json.dumps(dict(dn, metric="decode step through materialised bf16 weights",
                                  n_gpus=world, steps=args.steps, warmup=args.warmup,
                                  data="synthetic", config=workload_config(args))))
        return
    if args.mode == "prefill":
        pf = run_prefill(args, local_rank)
        if rank == 0:
            print(json.dumps(dict(pf, n_gpus=world, steps=args.steps, warmup=args.warmup,
                                  higher_is_better=True, data="synthetic")))
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()
        return
    # CPU baseline first (before any CUDA work), rank 0 at N = 1 only
    cpu = None
    if world == 1 and rank == 0 and not args.no_cpu_baseline:
        cpu = cpu_baseline(args.cpu_seconds, args.batch)
    r = run_bisco(args, rank, world, local_rank)
    subs, dense_cmp, prefill = {}, None, None
    if args.mode in ("both", "stack") and world == 1:
        import torch
        dev = torch.device("cuda", local_rank)
        subs = run_sweeps(args, r["stack"], r["stream"], dev)
        prefill = run_prefill_stack(args, r["stack"], r["stream"], dev)
        dense_cmp = run_dense_stack(args, r["stack"], r["stream"], dev)
        subs["residual_decode"] = run_residual_decode(args, r["stack"], r["stream"], dev)
        dense_cmp["fused_over_dense_batch1"] = (r["tokens_per_s"] / (args.batch / (dense_cmp["batch_1"]["ms_per_step"] * 1e-3))
                                                if args.batch == 1 else None)
    if rank == 0:
        line = {
            "metric": METRIC, "value": r["value"], "unit": "GB/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": r["ms_per_step"],
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f16", "data": "synthetic", "config": workload_config(args),
            "tokens_per_s": r["tokens_per_s"], "bytes_per_step": r["bytes_per_step"],
            "e2e": {"value": r["e2e_gbs"], "unit": "GB/s",
                    "h2d_bytes_per_step": r["h2d"], "d2h_bytes_per_step": r["d2h"],
                    "how": "pinned H2D of the step's activations + CUDA graph of the step's "
                           "4 calls per layer (bisco_gemv_multi q/k/v, bisco_gemv o, "
                           "bisco_gemv_multi gate/up, bisco_gemv down) + D2H of all outputs, "
                           "per step",
                    "ms_per_step": r["ms_e2e"]},
            "gpu_launches": r["launches"] * args.steps,
            "roofline": r["roofline"],
            "per_call": r["per_call"],
            "clocks": r["clocks"],
            "cpu_baseline": cpu,
            "parallelism": "replicas" if world > 1 else "single GPU",
            "prefill": prefill,
            "dense_comparison": dense_cmp,
        }
        line.update(subs)
        print(json.dumps(line))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
