#!/usr/bin/env python
"""Benchmark: the LLaMA-2-7B projection stack in decode (32 layers, 4/8-bit activations
by the layer mask {0, 1, 30, 31}), through the libdptq C ABI on one GB300.

A step is one pass of the whole hot path over one batch of M tokens: for every layer,
rotate + quantize the qkv input and run the q|k|v GEMM, then o, gate|up and down
(4 quantizations and 4 GEMMs per layer, 256 kernels per step), replayed as a CUDA
graph.  The packed weights (3.2 GB) exceed L2, so every step streams them from HBM.

Prints one JSON line (rank 0).  `--impl reference` times the CPU oracle instead on a
bounded sample of the same workload.  Under torchrun every rank runs an independent
replica (no collective on the data path); `value` is tokens over all ranks divided by
the slowest rank's time.
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

METRIC = "qlinear TOPS & HBM GB/s (% roofline); 32-layer projection-stack tokens/s"
UNIT = "tokens/s"
DEFAULT_M = 32


# ------------------------------------------------------------------------------ distributed
def dist_env():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)), int(os.environ.get("LOCAL_RANK", 0))


def init_dist(backend):
    import torch.distributed as dist
    rank, world, _ = dist_env()
    if world > 1 and not dist.is_initialized():
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group(backend=backend, rank=rank, world_size=world)
    return rank, world


def max_over_ranks(value: float, world: int, device=None) -> float:
    """Maximum of a per-rank float over all ranks (identity when world == 1)."""
    if world == 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def aggregate_value(tokens_per_rank: int, world: int, t_max_s: float) -> float:
    """Whole-job throughput: tokens of all ranks over the slowest rank's time."""
    return tokens_per_rank * world / t_max_s


# ------------------------------------------------------------------------------ clocks
REASONS = {0x1: "gpu_idle", 0x2: "applications_clocks_setting", 0x4: "sw_power_cap", 0x8: "hw_slowdown",
           0x10: "sync_boost", 0x20: "sw_thermal_slowdown", 0x40: "hw_thermal_slowdown",
           0x80: "hw_power_brake_slowdown", 0x100: "display_clock_setting"}


class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons during the timed region."""

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=clocks.sm,clocks.max.sm,clocks_event_reasons.active",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except (OSError, ValueError):
            self.proc = None
        return self

    def _read(self):
        for ln in self.proc.stdout:
            self.lines.append(ln.strip())

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.25)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], None, set()
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 3:
                continue
            try:
                sm.append(float(parts[0]))
                mx = float(parts[1])
                bits = int(parts[2], 16)
            except ValueError:
                continue
            for b, name in REASONS.items():
                if bits & b and name != "gpu_idle":
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": mx, "reasons": ["unsampled"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": len(sm)}


# ------------------------------------------------------------------------------ workload
def stack_groups(wl):
    """(name, K, N, had_block) per activation group of a layer: q|k|v, o, gate|up, down."""
    out = []
    for gname, projs in wl.groups():
        out.append((gname, projs[0].K, sum(p.N for p in projs), projs[0].had_block, [p for p in projs]))
    return out


def build_stack(dp, wl, device):
    """Pack every layer's weights (seeded, generated on the device) into library handles."""
    import torch
    names = [p.name for p in wl.projs]
    layers = []
    for layer in range(wl.layers):
        hs = []
        for gname, K, N, B, projs in stack_groups(wl):
            W = torch.cat([_inputs().torch_weights(p.N, p.K, layer, names.index(p.name), device) for p in projs])
            hs.append(dp.dptq_pack_weights(W.contiguous(), B))
            del W
        layers.append(hs)
    torch.cuda.synchronize()
    return layers


def _inputs():
    from paper_2606_12487_gb300 import inputs
    return inputs


class Stack:
    def __init__(self, dp, wl, layers, M, device, path="fused"):
        import torch
        self.dp, self.wl, self.layers, self.M = dp, wl, layers, M
        self.path = path   # "fused": one dptq_qlinear launch per projection; "split": quantize + GEMM
        groups = stack_groups(wl)
        self.x = [torch.from_numpy(_inputs().activations(wl, M, K, seed=gi)).to(device)
                  for gi, (_, K, _, _, _) in enumerate(groups)]
        self.out = [torch.empty((M, N), dtype=torch.float16, device=device) for (_, _, N, _, _) in groups]
        self.groups = groups

    def run(self, stream, gemm_events=None):
        """One step (the 32-layer stack).  With gemm_events, record an event pair around
        every GEMM launch (no graph)."""
        dp = self.dp
        for li, hs in enumerate(self.layers):
            bits = self.wl.bits(li)
            for gi, h in enumerate(hs):
                if self.path == "fused":
                    if gemm_events is not None:
                        e0, e1 = gemm_events.pop()
                        e0.record(stream)
                    dp.dptq_qlinear(h, self.x[gi], bits, self.out[gi], stream=stream)
                    if gemm_events is not None:
                        e1.record(stream)
                        gemm_events_done.append((e0, e1, self.gemm_bytes(gi, bits), self.gemm_ops(gi)))
                    continue
                dp.dptq_qlinear_quantize(h, self.x[gi], bits, stream=stream)
                if gemm_events is not None:
                    e0, e1 = gemm_events.pop()
                    e0.record(stream)
                    dp.dptq_qlinear_gemm(h, self.M, bits, self.out[gi], stream=stream)
                    e1.record(stream)
                    gemm_events_done.append((e0, e1, self.gemm_bytes(gi, bits), self.gemm_ops(gi)))
                else:
                    dp.dptq_qlinear_gemm(h, self.M, bits, self.out[gi], stream=stream)

    def gemm_bytes(self, gi, bits):
        """Algorithmic HBM bytes of one timed launch: packed int4 weights, weight scales and
        the fp16 output, plus the fp16 activations (fused launch) or the activation codes
        at b bits and token scales (GEMM launch of the split path)."""
        _, K, N, _, _ = self.groups[gi]
        M = self.M
        act = 2 * M * K if self.path == "fused" else M * K * bits // 8 + 4 * M
        return N * K // 2 + 4 * N + act + 2 * M * N

    def gemm_ops(self, gi):
        _, K, N, _, _ = self.groups[gi]
        return 2 * self.M * N * K

    def step_launches(self):
        """Kernel launches of one step: dptq_qlinear is one launch up to 64 tokens (fused)
        and two above (rotate-quantize, then GEMM); the split path is always two."""
        per = 1 if (self.path == "fused" and self.M <= 64) else 2
        return per * len(self.groups) * len(self.layers)

    def h2d_bytes(self):
        return sum(x.numel() * 2 for x in self.x)

    def d2h_bytes(self):
        return self.out[-1].numel() * 2


gemm_events_done = []


def kernel_source_sha():
    """sha256/16 of the sources the timed kernel is compiled from."""
    import hashlib
    h = hashlib.sha256()
    for f in ("qgemm.cu", "rotate_row.cuh", "dptq_device.cuh"):
        try:
            h.update(open(os.path.join(ROOT, "paper_2606_12487_gb300", "csrc", f), "rb").read())
        except OSError:
            return None
    return h.hexdigest()[:16]


def traffic_record(path_name):
    """DRAM bytes / algorithmic bytes of the timed kernel from the committed ncu summary,
    if the summary was taken on the current kernel sources and launch path (else None)."""
    import glob
    sha = kernel_source_sha()
    if sha is None:
        return None
    for path in sorted(glob.glob(os.path.join(ROOT, "profiles", "*.md"))):
        for ln in open(path):
            if ln.startswith("traffic_record:") and f"sha256/16={sha}" in ln and f"path={path_name}" in ln:
                kv = dict(p.split("=", 1) for p in ln.split() if "=" in p)
                return int(kv["dram_bytes"]) / int(kv["algorithmic_bytes"]), os.path.basename(path)
    return None


def time_graph(g, stream, steps, warmup, world, device_index, sample_clocks=True):
    import torch
    with torch.cuda.stream(stream):
        for _ in range(warmup):
            g.replay()
    torch.cuda.synchronize()
    barrier(world)
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    sampler = ClockSampler(device_index) if sample_clocks else None
    if sampler:
        sampler.__enter__()
    with torch.cuda.stream(stream):
        e0.record(stream)
        for _ in range(steps):
            g.replay()
        e1.record(stream)
    torch.cuda.synchronize()
    if sampler:
        sampler.__exit__(None, None, None)
    barrier(world)
    ms = e0.elapsed_time(e1) / steps
    return ms, (sampler.summary() if sampler else None)


class EagerStep:
    """Stands in for a captured graph: replay() launches the step's kernels directly."""

    def __init__(self, stack, stream):
        self.stack, self.stream = stack, stream

    def replay(self):
        self.stack.run(self.stream)


def capture(stack, stream, eager=False):
    import torch
    if eager:
        return EagerStep(stack, stream)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        stack.run(stream)
    torch.cuda.synchronize()
    return g


def measure_gemm_kernels(stack, stream):
    """Per-launch CUDA-event durations of every GEMM of one eager step (after one warm
    eager step).  Returns (algorithmic bytes, ops, seconds) summed over the launches."""
    import torch
    stack.run(stream)
    torch.cuda.synchronize()
    n = len(stack.layers) * len(stack.groups)
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
    gemm_events_done.clear()
    stack.run(stream, gemm_events=list(reversed(evs)))
    torch.cuda.synchronize()
    tb = to = tt = 0.0
    per = []
    for e0, e1, b, o in gemm_events_done:
        t = e0.elapsed_time(e1) / 1e3
        tb += b
        to += o
        tt += t
        per.append(t)
    return tb, to, tt, n


def e2e_measure(stack, g, stream, steps, world):
    """Same metric through the public API with host buffers: per step, H2D copies of
    the step's inputs from pinned memory, the stack as the user calls it (every
    projection a dptq_qlinear call through the C ABI, launched eagerly, no graph), and a
    D2H read of the result."""
    import torch
    hx = [x.cpu().pin_memory() for x in stack.x]
    hout = torch.empty(stack.out[-1].shape, dtype=torch.float16).pin_memory()
    for _ in range(3):
        with torch.cuda.stream(stream):
            for h, d in zip(hx, stack.x):
                d.copy_(h, non_blocking=True)
            stack.run(stream)
            hout.copy_(stack.out[-1], non_blocking=True)
    torch.cuda.synchronize()
    barrier(world)
    t0 = time.perf_counter()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e0.record(stream)
        for _ in range(steps):
            for h, d in zip(hx, stack.x):
                d.copy_(h, non_blocking=True)
            stack.run(stream)
            hout.copy_(stack.out[-1], non_blocking=True)
        e1.record(stream)
    torch.cuda.synchronize()
    wall = time.perf_counter() - t0
    return max(e0.elapsed_time(e1) / 1e3, 0.0) / steps, wall / steps


# ------------------------------------------------------------------------------ per-shape kernels
L2_BYTES = 129 * 2 ** 20


def shape_cases():
    """(label, M, N, K, had_block, bits): the single 256 -> 512 linear, the LLaMA-2-7B
    decode projections, the LLaMA-3-8B and LLaMA-2-13B prefill ones and the LLaMA-2-70B
    ones at four token counts (q|k|v and gate|up as concatenated N), at A4 and, for the
    prefill shapes, A8."""
    d = [("7b qkv", 12288, 4096, 4096), ("7b o", 4096, 4096, 4096), ("7b gate|up", 22016, 4096, 4096),
         ("7b down", 4096, 11008, 256)]
    out = [("single linear 256->512", 16, 512, 256, 256, bits) for bits in (4, 8)]
    out += [(f"{n} decode", 32, N, K, B, 4) for n, N, K, B in d]
    out += [("7b gate|up decode", 32, 22016, 4096, 4096, 8), ("7b gate|up decode", 1, 22016, 4096, 4096, 4),
            ("7b gate|up decode", 8, 22016, 4096, 4096, 4)]
    p8 = [("8b q prefill", 4096, 4096), ("8b gate|up prefill", 28672, 4096), ("8b down prefill", 4096, 14336)]
    out += [(n, 2048, N, K, 2048, bits) for bits in (4, 8) for n, N, K in p8]
    # LLaMA-2-13B prefill (M = 4096, block Hadamard 1024; gate|up A8 as on its masked layers)
    p13 = [("13b qkv prefill", 15360, 5120), ("13b o prefill", 5120, 5120), ("13b gate|up prefill", 27648, 5120),
           ("13b down prefill", 5120, 13824)]
    out += [(n, 4096, N, K, 1024, 4) for n, N, K in p13] + [("13b gate|up prefill", 4096, 27648, 5120, 1024, 8)]
    # LLaMA-2-70B (block Hadamard 4096) at M = 1, 64, 512 and 8192 tokens
    p70 = [("70b qkv", 10240, 8192), ("70b o", 8192, 8192), ("70b gate|up", 57344, 8192), ("70b down", 8192, 28672)]
    out += [(n, M, N, K, 4096, 4) for M in (1, 64, 512, 8192) for n, N, K in p70]
    out += [("70b gate|up", 8192, 57344, 8192, 4096, 8)]
    return out


def run_shapes(args):
    """Times one launch of each shape (CUDA events over graph replays of 40 launches) with
    as many weight copies as make the rotation through them at least twice the L2, so
    every launch streams its weights from HBM."""
    import math
    import torch
    from paper_2606_12487_gb300 import dptq, inputs
    dptq.load()
    dev = torch.device("cuda")
    dptq.dptq_reserve(2048, 14336, 0)
    peaks = {}
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            peaks = json.load(f)
    except OSError:
        pass
    hbm = float(peaks.get("hbm_gbs", 6800.0))
    fp8 = 2.0 * float(peaks.get("bf16_tflops", 1900.0))
    stream = torch.cuda.Stream(device=dev)
    reps = 40

    def t_graph(fns):
        with torch.cuda.stream(stream):
            for f in fns[:3]:
                f()
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for i in range(reps):
                fns[i % len(fns)]()
        for _ in range(2):
            g.replay()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            e0.record(stream)
            g.replay()
            e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) * 1e3 / reps

    rows = []
    for label, M, N, K, B, bits in ([] if args.extra_only else shape_cases()):
        if args.only and args.only not in f"{label} M={M} A{bits}":
            continue
        wbytes = N * K // 2
        copies = max(1, min(64, math.ceil(2 * L2_BYTES / wbytes)))
        W = inputs.torch_weights(N, K, 0, 0, dev)
        hs = [dptq.dptq_pack_weights(W, B) for _ in range(copies)]
        del W
        x = torch.from_numpy(inputs.activations(inputs.llama2_7b_decode(), M, K)).to(dev)
        out = torch.empty((M, N), dtype=torch.float16, device=dev)
        s_ = stream
        t_q = t_graph([lambda h=h: dptq.dptq_qlinear_quantize(h, x, bits, stream=s_) for h in hs[:1]])
        with torch.cuda.stream(stream):
            dptq.dptq_qlinear_quantize(hs[0], x, bits, stream=s_)
        t_g = t_graph([lambda h=h: dptq.dptq_qlinear_gemm(h, M, bits, out, stream=s_) for h in hs])
        t_l = t_graph([lambda h=h: dptq.dptq_qlinear(h, x, bits, out, stream=s_) for h in hs])
        gemm_b = wbytes + 4 * N + M * K * bits // 8 + 4 * M + 2 * M * N
        ql_b = wbytes + 4 * N + 2 * M * K + 2 * M * N
        ops = 2 * M * N * K
        # rotate + quantize: the fp16 row in, b-bit codes and a scale out (algorithmic bytes;
        # the GEMM operand planes it actually writes hold one byte per code and plane)
        q_b = 2 * M * K + M * K * bits // 8 + 4 * M
        r = {"shape": label, "M": M, "N": N, "K": K, "had_block": B, "bits": bits, "weight_copies": copies,
             "quantize_us": t_q, "gemm_us": t_g, "qlinear_us": t_l, "quantize_gbs": q_b / t_q / 1e3,
             "quantize_hbm_frac": q_b / t_q / 1e3 / hbm,
             "gemm_gbs": gemm_b / t_g / 1e3, "qlinear_gbs": ql_b / t_l / 1e3,
             "gemm_tops": ops / t_g / 1e6, "qlinear_tops": ops / t_l / 1e6}
        if M <= 64:
            r["roofline"] = {"bound": "hbm", "peak_gbs": hbm, "gemm_frac": r["gemm_gbs"] / hbm,
                             "qlinear_frac": r["qlinear_gbs"] / hbm}
        else:
            r["roofline"] = {"bound": "tensor", "peak_tflops": fp8, "peak_note": "2 x bf16 burst measured (fp8 nominal ratio)",
                             "gemm_frac": r["gemm_tops"] / fp8, "qlinear_frac": r["qlinear_tops"] / fp8}
        rows.append(r)
        print(f"[shapes] {label} M={M} A{bits}: quantize {t_q:.1f} us, gemm {t_g:.1f} us, qlinear {t_l:.1f} us",
              file=sys.stderr, flush=True)
        for h in hs:
            h.close()
        del hs
        torch.cuda.synchronize()
    # KV4 group-128 quantizer over one layer's K cache (LLaMA-2-7B, 32 heads x 128, 8192
    # tokens: 64 MB fp16) and the sensitivity policy over 32 layers x 512 tokens x 4096
    # (2 x 268 MB fp32): both HBM-bound; inputs rotated through copies beyond 2x L2.
    extra = []
    T, H, D = 8192, 32, 128
    kvs = [torch.from_numpy(inputs.activations(inputs.llama2_7b_decode(), 1024, 128)).to(dev).repeat(T * H // 1024, 1)
           for _ in range(3)]
    codes = torch.empty((T * H, D // 2), dtype=torch.uint8, device=dev)
    sc = torch.empty((T * H, 1), dtype=torch.float32, device=dev)
    t_kv = t_graph([lambda kv=kv: dptq.dptq_kv4_quantize(kv, 128, codes, sc, stream=stream) for kv in kvs])
    kv_b = T * H * D * 2 + T * H * D // 2 + T * H * 4
    extra.append({"kernel": "kv4_quantize", "rows": T * H, "cols": D, "group": 128, "us": t_kv,
                  "gbs": kv_b / t_kv / 1e3, "roofline": {"bound": "hbm", "peak_gbs": hbm, "frac": kv_b / t_kv / 1e3 / hbm}})
    del kvs, codes, sc
    L, TT, d = 32, 512, 4096
    g = torch.Generator(device=dev).manual_seed(9)
    xs = torch.randn((L, TT, d), generator=g, device=dev)
    dxs = 0.1 * torch.randn((L, TT, d), generator=g, device=dev)
    jr = torch.empty((L,), dtype=torch.float64, device=dev)
    snr = torch.empty((L,), dtype=torch.float64, device=dev)
    bo = torch.empty((L,), dtype=torch.uint8, device=dev)
    t_pol = t_graph([lambda: dptq.dptq_sensitivity_policy(xs, dxs, 4, 1e-6, 0.1, 20.0, jr, snr, bo, stream=stream)])
    pol_b = 2 * L * TT * d * 4
    extra.append({"kernel": "sensitivity_policy", "L": L, "T": TT, "d": d, "us": t_pol, "gbs": pol_b / t_pol / 1e3,
                  "roofline": {"bound": "hbm", "peak_gbs": hbm, "frac": pol_b / t_pol / 1e3 / hbm}})
    print(f"[shapes] kv4 {t_kv:.1f} us, policy {t_pol:.1f} us", file=sys.stderr, flush=True)
    dptq.dptq_last_device_error()
    print(json.dumps({"mode": "shapes", "timing": "CUDA events over graph replays, weights rotated through "
                                                  ">= 2x L2 of copies", "shapes": rows, "extra_kernels": extra}),
          flush=True)
    return 0


# ------------------------------------------------------------------------------ prefill stack
PREFILL_M = 2048


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f)
    except OSError:
        return {}


def measure_prefill(dptq, device, stream, steps, warmup, world, local):
    """The LLaMA-3-8B prefill projection stack: 32 layers at M = 2048 tokens with the
    seeded mask of 6 A8 layers; each projection group (q|k|v, o, gate|up, down) is one
    dptq_qlinear call, i.e. a rotate-quantize launch and a GEMM launch, and the step is
    replayed as a CUDA graph.  Inputs (16-59 MB per group) and weights (3.5 GB) exceed
    L2 between replays.  Returns the `prefill` object of the JSON line."""
    import torch
    from paper_2606_12487_gb300 import inputs
    wl = inputs.llama3_8b_prefill()
    M = PREFILL_M
    layers = build_stack(dptq, wl, device)
    max_k = max(K for _, K, _, _, _ in stack_groups(wl))
    dptq.dptq_reserve(M, max_k, 0)
    stack = Stack(dptq, wl, layers, M, device, "fused")
    g = capture(stack, stream)
    ms, clocks = time_graph(g, stream, steps, warmup, world, local)
    ms = max_over_ranks(ms, world, device)
    ops = sum(2 * M * N * K for _, K, N, _, _ in stack.groups) * len(layers)
    # One eager step with CUDA events around every launch (on the launching stream): the
    # GEMM launches and the rotate-quantize launches, timed apart.
    dptq.dptq_qlinear_quantize(layers[0][0], stack.x[0], 4, stream=stream)
    torch.cuda.synchronize()
    t_q = t_g = 0.0
    gemm_ops = 0
    evs = []
    with torch.cuda.stream(stream):
        for li, hs in enumerate(layers):
            bits = wl.bits(li)
            for gi, h in enumerate(hs):
                e = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
                e[0].record(stream)
                dptq.dptq_qlinear_quantize(h, stack.x[gi], bits, stream=stream)
                e[1].record(stream)
                dptq.dptq_qlinear_gemm(h, M, bits, stack.out[gi], stream=stream)
                e[2].record(stream)
                _, K, N, _, _ = stack.groups[gi]
                evs.append((e, 2 * M * N * K))
    torch.cuda.synchronize()
    for e, o in evs:
        t_q += e[0].elapsed_time(e[1]) / 1e3
        t_g += e[1].elapsed_time(e[2]) / 1e3
        gemm_ops += o
    peaks = load_peaks()
    bf16_sus = float(peaks.get("bf16_tflops_sustained", 1700.0))
    bf16_burst = float(peaks.get("bf16_tflops", 1900.0))
    fp8_sus, fp8_burst = 2.0 * bf16_sus, 2.0 * bf16_burst
    n_gemm = len(evs)
    gemm_tops = gemm_ops / t_g / 1e12
    stack_tops = ops / (ms / 1e3) / 1e12
    rot_bytes = sum(M * K * 2 + M * K * wl.bits(li) // 8 + 4 * M
                    for li in range(len(layers)) for _, K, _, _, _ in stack.groups)
    hbm = float(peaks.get("hbm_gbs", 6800.0))
    del g
    out = {
        "workload": f"llama3-8b prefill projection stack, {len(layers)} layers, M={M} tokens, "
                    f"A8 on layers {list(wl.mask_a8)}, block Hadamard 2048",
        "tokens_per_s": aggregate_value(M, world, ms / 1e3), "ms_per_step": ms, "steps": steps, "warmup": warmup,
        "effective_tops": stack_tops, "ops_per_step": ops,
        "ops_note": "2*M*N*K effective integer ops per projection (A8 layers issue twice the MMA work)",
        "gpu_launches": stack.step_launches() * steps,
        "roofline": {"bound": "tensor", "achieved": stack_tops, "peak": fp8_sus, "unit": "TFLOP/s",
                     "frac": stack_tops / fp8_sus,
                     "peak_source": "2 x MEASURED_PEAKS.json bf16_tflops_sustained (fp8 = 2 x bf16 nominal ratio)",
                     "achieved_note": "effective ops of the step / graph-replay step time (both launches of every "
                                      "projection)",
                     "gemm_kernel": {"kernel": "qgemm_kernel (192-token tiles A4, 128-token tiles A8)",
                                     "achieved_tflops": gemm_tops, "peak": fp8_burst,
                                     "frac": gemm_tops / fp8_burst, "launches": n_gemm,
                                     "avg_launch_us": t_g / n_gemm * 1e6,
                                     "note": "eager pass, CUDA events around each GEMM launch on its stream; "
                                             "peak = 2 x bf16 burst"}},
        "time_shares": {"gemm": t_g / (t_g + t_q), "rotate_quantize": t_q / (t_g + t_q)},
        "rotate_quantize": {"us_per_step": t_q * 1e6, "gbs": rot_bytes / t_q / 1e9,
                            "hbm_frac": rot_bytes / t_q / 1e9 / hbm,
                            "bytes_note": "2MK (fp16 in) + MK b/8 (codes) + 4M (scales) per launch"},
        "clocks": clocks,
    }
    for hs in layers:
        for h in hs:
            h.close()
    del stack, layers
    torch.cuda.synchronize()
    return out


# ------------------------------------------------------------------------------ oracle timing
def oracle_sample_times(wl, budget_s: float, tokens: int = 1):
    """Time the oracle's online path (rotate + quantize, int GEMM, epilogue) per layer
    group at each bit width on `tokens` tokens.  Weight codes are seeded random int4
    values (packing is offline and not part of the timed path).  Returns
    {(group, bits): seconds per call} and the number of timed calls."""
    import numpy as np

    import oracle
    inputs = _inputs()
    groups = stack_groups(wl)
    data = {}
    for gi, (gname, K, N, B, _) in enumerate(groups):
        q = inputs.random_codes(N, K, 4, seed=100 + gi)
        sw = np.full((N,), 0.001, dtype=np.float32)
        x = inputs.activations(wl, tokens, K, seed=gi)
        data[gi] = (x, B, q, sw)
    times = {}
    calls = 0
    t_start = time.perf_counter()
    while True:
        for gi in data:
            for bits in (4, 8):
                x, B, q, sw = data[gi]
                t0 = time.perf_counter()
                oracle.qlinear(x, B, bits, q, sw)
                times.setdefault((gi, bits), []).append(time.perf_counter() - t0)
                calls += 1
        if time.perf_counter() - t_start >= budget_s:
            break
    return {k: statistics.median(v) for k, v in times.items()}, calls


def stack_time_from(wl, times):
    n_groups = len(stack_groups(wl))
    return sum(times[(gi, wl.bits(li))] for li in range(wl.layers) for gi in range(n_groups))


def cpu_baseline(wl, budget_s=12.0, all_cores_budget_s=6.0):
    times, calls = oracle_sample_times(wl, budget_s)
    t_stack = stack_time_from(wl, times)
    line = {"value": 1.0 / t_stack, "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": f"1 token through each of the 4 projection groups at 4 and 8 bits ({calls} oracle calls, "
                      f"~{budget_s:.0f} s), weights as random int4 codes; 32-layer stack time summed from the "
                      "per-group medians with the layer mask",
            "host": host_cpu()}
    try:
        line["all_cores"] = cpu_baseline_all_cores(wl, all_cores_budget_s)
    except Exception as e:   # the single-core figure stands on its own
        line["all_cores"] = {"unavailable": f"{type(e).__name__}: {e}"}
    return line


def host_cpu():
    """Core count and CPU model of this host (the model line of /proc/cpuinfo where present)."""
    import platform
    model = None
    try:
        with open("/proc/cpuinfo") as f:
            for ln in f:
                key = ln.split(":", 1)[0].strip().lower()
                if key in ("model name", "cpu model", "hardware") and ":" in ln:
                    model = ln.split(":", 1)[1].strip()
                    break
    except OSError:
        pass
    return {"nproc": usable_cores(), "machine": platform.machine(), "cpu_model": model or platform.processor() or None}


def usable_cores():
    """Cores this process may run on (its affinity set; the machine's count as a fallback)."""
    try:
        return len(os.sched_getaffinity(0))
    except (AttributeError, OSError):
        return os.cpu_count() or 1


def _oracle_worker(budget_s):
    """One process of the all-cores oracle timing: the single-core sample, returned as the
    stack time of one token stream."""
    wl = _inputs().llama2_7b_decode()
    times, calls = oracle_sample_times(wl, budget_s)
    return stack_time_from(wl, times), calls


def cpu_baseline_all_cores(wl, budget_s):
    """The same oracle sample in one process per core at once (spawned, so no CUDA state is
    inherited): independent token streams, tokens/s summed over the processes."""
    import multiprocessing as mp
    n = min(64, usable_cores())
    with mp.get_context("spawn").Pool(n) as pool:
        res = pool.map(_oracle_worker, [budget_s] * n)
    return {"value": sum(1.0 / t for t, _ in res), "unit": UNIT, "cores": n,
            "sample": f"{n} processes, each the single-core sample for ~{budget_s:.0f} s "
                      f"({sum(c for _, c in res)} oracle calls in all); one token stream per process"}


def run_reference(args):
    rank, world, _ = dist_env()
    if world > 1 and rank != 0:
        return 0
    from paper_2606_12487_gb300 import inputs
    wl = inputs.llama2_7b_decode()
    # Each step: the oracle on one projection group of one layer for one token, cycling
    # through the stack; the stack time is assembled from the per-(group, bits) medians.
    groups = stack_groups(wl)
    import numpy as np

    import oracle
    data = []
    for gi, (gname, K, N, B, _) in enumerate(groups):
        data.append((inputs.activations(wl, 1, K, seed=gi), B, inputs.random_codes(N, K, 4, seed=100 + gi),
                     np.full((N,), 0.001, dtype=np.float32)))
    order = [(li, gi) for li in range(wl.layers) for gi in range(len(groups))]
    times = {}
    t_steps = []
    for i in range(args.warmup + args.steps):
        li, gi = order[i % len(order)]
        bits = wl.bits(li)
        x, B, q, sw = data[gi]
        t0 = time.perf_counter()
        oracle.qlinear(x, B, bits, q, sw)
        dt = time.perf_counter() - t0
        if i >= args.warmup:
            times.setdefault((gi, bits), []).append(dt)
            t_steps.append(dt)
    for gi in range(len(groups)):
        for bits in (4, 8):
            if (gi, bits) not in times:
                x, B, q, sw = data[gi]
                t0 = time.perf_counter()
                oracle.qlinear(x, B, bits, q, sw)
                times[(gi, bits)] = [time.perf_counter() - t0]
    med = {k: statistics.median(v) for k, v in times.items()}
    t_stack = stack_time_from(wl, med)
    value = 1.0 / t_stack
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * statistics.mean(t_steps),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": "llama2-7b decode projection stack, 32 layers, A8 mask {0,1,30,31}, "
                               "oracle sample of 1 token per step (one projection group per step)",
                   "global_batch": 1, "parallelism": "replicas"},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle",
                         "sample": "1 token, one projection group per step cycling through the stack; "
                                   "stack time from per-(group, bits) medians"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------------------------------------ main
def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="dptq", choices=["dptq", "reference"])
    ap.add_argument("--m", type=int, default=DEFAULT_M, help="tokens per step (decode batch)")
    ap.add_argument("--sweep", default="1,8", help="extra token counts measured for the m_sweep entry")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--eager", action="store_true",
                    help="launch the step's kernels directly instead of replaying a CUDA graph")
    ap.add_argument("--path", default="fused", choices=["fused", "split"],
                    help="fused: one launch per projection (rotation + quantization + GEMM); "
                         "split: rotate-quantize launch, then GEMM launch")
    ap.add_argument("--layers", type=int, default=0,
                    help="run only the first L layers (small cases for profiler captures; 0 = all)")
    ap.add_argument("--shapes", action="store_true",
                    help="time each decode / prefill projection shape alone and print one JSON line of them")
    ap.add_argument("--extra-only", action="store_true",
                    help="with --shapes: time only the KV4 quantizer and the sensitivity policy")
    ap.add_argument("--prefill-steps", type=int, default=10,
                    help="timed steps of the LLaMA-3-8B prefill stack (the `prefill` object; 0 = skip it)")
    ap.add_argument("--only", default="",
                    help="with --shapes: only the shapes whose label 'NAME M=.. A..' contains this text "
                         "(the KV4 and policy timings still follow)")
    args = ap.parse_args(argv)
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        return run_reference(args)
    if args.shapes:
        return run_shapes(args)

    import torch
    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    rank, world = init_dist("nccl")
    from paper_2606_12487_gb300 import dptq, inputs
    dptq.load()
    wl = inputs.llama2_7b_decode()
    if args.layers:
        wl.layers = min(args.layers, wl.layers)
    print(f"[bench] rank {rank}/{world}: packing {wl.layers}-layer stack", file=sys.stderr, flush=True)
    layers = build_stack(dptq, wl, device)
    max_k = max(K for _, K, _, _, _ in stack_groups(wl))
    max_m = max([args.m] + [int(v) for v in args.sweep.split(",") if v])
    dptq.dptq_reserve(max_m, max_k, 0)
    stream = torch.cuda.Stream(device=device)

    stack = Stack(dptq, wl, layers, args.m, device, args.path)
    g = capture(stack, stream, args.eager)
    ms, clocks = time_graph(g, stream, args.steps, args.warmup, world, local)
    ms_max = max_over_ranks(ms, world, device)
    value = aggregate_value(args.m, world, ms_max / 1e3)

    tb, to, tt, n_gemm = measure_gemm_kernels(stack, stream)
    n_launches_step = stack.step_launches()
    h2d_bytes, d2h_bytes = stack.h2d_bytes(), stack.d2h_bytes()
    peaks = load_peaks()
    hbm_peak = float(peaks.get("hbm_gbs", 6800.0))
    # The timed step is nothing but the n_gemm launches of this kernel, back to back, so
    # its average launch duration over the timed region is the step time / n_gemm and the
    # achieved rate is the step's algorithmic bytes / the step time.  The eager pass with
    # events around each launch (no graph, no overlap between launches) is reported beside it.
    achieved = tb / (ms_max / 1e3) / 1e9
    isolated = tb / tt / 1e9
    rec = traffic_record(args.path)
    traffic = rec[0] * tb / n_gemm if rec else None
    e2e_dev_s, e2e_wall_s = e2e_measure(stack, g, stream, max(10, args.steps // 4), world)
    e2e_s = max_over_ranks(e2e_dev_s, world, device)

    sweep = {}
    for m in [int(v) for v in args.sweep.split(",") if v]:
        st = Stack(dptq, wl, layers, m, device, args.path)
        gm = capture(st, stream, args.eager)
        ms_m, _ = time_graph(gm, stream, max(20, args.steps // 2), args.warmup, world, local, sample_clocks=False)
        ms_m = max_over_ranks(ms_m, world, device)
        tbm, _, ttm, _ = measure_gemm_kernels(st, stream)
        sweep[str(m)] = {"tokens_per_s": aggregate_value(m, world, ms_m / 1e3), "ms_per_step": ms_m,
                         "gemm_gbs": tbm / (ms_m / 1e3) / 1e9, "isolated_launch_gbs": tbm / ttm / 1e9}
        del gm, st
    sweep[str(args.m)] = {"tokens_per_s": value, "ms_per_step": ms_max, "gemm_gbs": achieved,
                          "isolated_launch_gbs": isolated}

    # Free the decode stack before the prefill stack is packed.
    del g, stack
    for hs in layers:
        for h in hs:
            h.close()
    torch.cuda.synchronize()
    prefill = None
    if args.prefill_steps > 0 and not args.layers:
        print(f"[bench] rank {rank}/{world}: prefill stack", file=sys.stderr, flush=True)
        prefill = measure_prefill(dptq, device, stream, args.prefill_steps, args.warmup, world, local)

    dptq.dptq_last_device_error()
    if rank != 0:
        return 0
    cpu = None if args.no_cpu_baseline or world > 1 else cpu_baseline(inputs.llama2_7b_decode())
    weight_bytes = sum(N * K // 2 for _, K, N, _, _ in stack_groups(wl)) * wl.layers
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_max, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "int4xint4/int8 (fp8-e4m3 tensor cores, exact int32)", "data": "synthetic",
        "config": {"workload": f"llama2-7b decode projection stack, {wl.layers} layers, M={args.m} tokens, "
                               "A8 on layers {0,1,30,31}", "global_batch": args.m * world, "seq_len": 1,
                   "parallelism": f"replicas x{world}", "l2": "weights 3.24 GB > L2 (streamed every step)",
                   "path": args.path,
                   "weight_bytes_per_step": weight_bytes},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": hbm_peak, "unit": "GB/s",
                     "frac": achieved / hbm_peak, "traffic": traffic,
                     "kernel": "qgemm_kernel (fused rotation + quantization + GEMM)" if args.path == "fused"
                               else "qgemm_kernel",
                     "traffic_note": (f"bytes per average launch: ncu DRAM/algorithmic ratio {rec[0]:.3f} "
                                      f"({rec[1]}) x {tb / n_gemm:.0f} algorithmic bytes") if rec else
                                     "no capture of the current kernel source",
                     "peak_source": "MEASURED_PEAKS.json hbm_gbs (copy, burst)",
                     "launches_per_step": n_gemm,
                     "avg_launch_us": ms_max * 1e3 / n_gemm,
                     "achieved_note": "algorithmic bytes of the step's launches / timed step (graph replay)",
                     "isolated_launch_gbs": isolated},
        "gemm_tops": to / (ms_max / 1e3) / 1e12,
        "stack_weight_gbs": weight_bytes / (ms_max / 1e3) / 1e9,
        "m_sweep": sweep,
        "e2e": {"value": aggregate_value(args.m, world, e2e_s), "unit": UNIT,
                "h2d_bytes_per_step": h2d_bytes, "d2h_bytes_per_step": d2h_bytes,
                "wall_ms_per_step": e2e_wall_s * 1e3},
        "gpu_launches": n_launches_step * args.steps,
        "clocks": clocks,
        "cpu_baseline": cpu,
        "prefill": prefill,
    }
    print(json.dumps(line), flush=True)
    return 0


if __name__ == "__main__":
    sys.exit(main())
