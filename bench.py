"""Benchmark of the MoE decode layer on GB300.

python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                [--workload NAME] [--tokens T]

One step = one decode layer (router GEMV + top-k + permute + gate/up SwiGLU
+ down + combine) over a batch of T tokens, on synthetic seeded inputs shaped
like the Qwen3-235B-A22B NVFP4 MoE layer (H=4096, E=128, top-8, I=1536) at
T=64 by default.  The metric is decode-layer tokens/s; achieved HBM GB/s, the
roofline fraction of the dominant kernel and J/token (NVML energy counter)
are reported beside it.  Under torchrun each rank runs an independent replica
on its own GPU (the layer does not shard across GPUs); the timed region is
bracketed by a barrier and the slowest rank's time is reported.

--impl reference times the float64 CPU oracle (the reference semantics) on
the host cores on a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import ctypes
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

WORKLOADS = {
    # name: (fmt, H, E, k, I)
    "qwen3_235b_nvfp4": (2, 4096, 128, 8, 1536),
    "qwen3_480b_fp8": (1, 6144, 160, 8, 2560),
    "tiny_fp8": (1, 512, 8, 2, 256),
}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="qwen3_235b_nvfp4", choices=sorted(WORKLOADS))
    ap.add_argument("--tokens", type=int, default=64)
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-energy", action="store_true")
    return ap.parse_args()


# ---------------------------------------------------------------- distributed
def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def barrier_max(value, world):
    """Barrier, then the maximum of `value` over ranks."""
    if world == 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device="cuda")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


# ---------------------------------------------------------------- clocks / energy
class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during a region."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "20"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except (OSError, ValueError):
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, smax, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [v.strip() for v in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax = float(f[2])
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": smax,
                "reasons": sorted(reasons), "samples": len(sm)}


class Nvml:
    """Total-energy counter of one GPU through libnvidia-ml (read only)."""

    def __init__(self, index):
        self.ok = False
        try:
            self.lib = ctypes.CDLL("libnvidia-ml.so.1")
            if self.lib.nvmlInit_v2() != 0:
                return
            self.h = ctypes.c_void_p()
            if self.lib.nvmlDeviceGetHandleByIndex_v2(index, ctypes.byref(self.h)) != 0:
                return
            self.ok = self.energy_mj() is not None
        except OSError:
            pass

    def energy_mj(self):
        v = ctypes.c_ulonglong(0)
        if self.lib.nvmlDeviceGetTotalEnergyConsumption(self.h, ctypes.byref(v)) != 0:
            return None
        return v.value


# ---------------------------------------------------------------- CPU oracle
def _oracle_weights(w):
    from oracle import oracle
    return oracle.ExpertWeights(w.fmt, w.E, w.H, w.I, *[
        None if t is None else t.detach().cpu().numpy()
        for t in (w.w_gate, w.w_up, w.w_down, w.s_gate, w.s_up, w.s_down, w.ts_gate, w.ts_up,
                  w.ts_down)])


class OracleSample:
    """The float64 oracle (router + top-k + experts + combine) on the first n
    tokens of the workload batch, on the host cores.  n is chosen so that one
    pass takes about `budget_s` seconds; only the experts those tokens route
    to are generated (on the host, untimed) unless the full weights are given."""

    def __init__(self, fmt, H, E, k, I, T, seed, budget_s=10.0, w=None):
        import numpy as np
        import torch

        from oracle import oracle
        from paper_2609_11133_gb300 import synth
        self.k = k
        self.cores = len(os.sched_getaffinity(0))
        x = synth.make_x(T, H, seed=seed)
        self.xb = x.view(torch.int16).numpy().view(np.uint16)
        self.wr = synth.make_router(E, H, seed=seed).numpy()
        ids, _ = oracle.topk(oracle.router_logits(self.xb, self.wr), k)
        # calibrate on one token
        if w is None:
            w = synth.make_weights(fmt, E, H, I, seed=seed, experts=np.unique(ids[:1]))
        self.ow = _oracle_weights(w)
        self.n = 1
        dt = self.run()
        n = max(1, min(T, int(budget_s / max(dt, 1e-3))))
        self.n = n
        if n > 1 and not self._full(w, E):
            w = synth.make_weights(fmt, E, H, I, seed=seed, experts=np.unique(ids[:n]))
            self.ow = _oracle_weights(w)
        self.experts = int(np.unique(ids[:n]).size)

    @staticmethod
    def _full(w, E):
        return bool((w.w_gate.reshape(E, -1)[:, :64] != 0).any(dim=1).all())

    def run(self):
        from oracle import oracle
        sub = self.xb[:self.n]
        t0 = time.perf_counter()
        ids, gates = oracle.topk(oracle.router_logits(sub, self.wr), self.k)
        oracle.moe_tokens(self.ow, sub, ids, gates)
        return time.perf_counter() - t0


def cpu_oracle_sample(fmt, H, E, k, I, T, seed, w=None, budget_s=10.0):
    s = OracleSample(fmt, H, E, k, I, T, seed, budget_s=budget_s, w=w)
    dt = s.run()
    return {"value": s.n / dt, "unit": "tokens/s", "cores": s.cores, "kind": "oracle",
            "sample": f"first {s.n} of {T} tokens ({s.experts} experts): router, top-k, "
                      f"experts and combine in float64, {dt:.2f} s"}


def layer_bytes(fmt, H, E, k, I, T, n_active, w_expert_bytes, router_bytes):
    act = 2 * T * H * 2  # x in, out
    return router_bytes + n_active * w_expert_bytes + act


# ---------------------------------------------------------------- our arm
def run_ours(args):
    import numpy as np
    import torch

    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    else:
        torch.cuda.set_device(0)
    from paper_2609_11133_gb300 import binding, synth

    fmt, H, E, k, I = WORKLOADS[args.workload]
    T = args.tokens
    dev = "cuda"
    w = synth.make_weights(fmt, E, H, I, seed=args.seed, device=dev)
    x = synth.make_x(T, H, seed=args.seed + rank, device=dev)
    wr = synth.make_router(E, H, seed=args.seed, device=dev)
    out = torch.empty((T, H), dtype=torch.bfloat16, device=dev)
    ws = binding.alloc_workspace(binding.moe_workspace_size(w, T, k))
    ids = torch.empty((T, k), dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream()

    # routing of this batch -> unique experts -> algorithmic bytes
    binding.moe_decode_layer_ex(x, wr, None, w, k, out, ws, topk_ids_out=ids)
    torch.cuda.synchronize()
    assert binding.moe_read_status(ws) == 0
    n_active = int(torch.unique(ids).numel())
    per_expert = w.nbytes_expert()
    gu_bytes = (w.w_gate[0].numel() + w.w_up[0].numel()) * 1 + \
        (w.s_gate[0].numel() * w.s_gate.element_size() + w.s_up[0].numel() * w.s_up.element_size())
    dn_bytes = w.w_down[0].numel() + w.s_down[0].numel() * w.s_down.element_size()
    if fmt == 2:
        gu_bytes += 8
        dn_bytes += 4
    router_bytes = E * H * 4
    B = layer_bytes(fmt, H, E, k, I, T, n_active, per_expert, router_bytes)

    ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]

    def step(record):
        binding.moe_decode_layer_ex(x, wr, None, w, k, out, ws, events=ev if record else None)

    for _ in range(max(3, args.warmup)):
        step(False)
    torch.cuda.synchronize()

    # One layer call captured in a CUDA graph: the timed loop replays it, so the
    # host's launch work is not part of the measurement (the layer takes no
    # host-side decisions between its kernels).
    g_step = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_step):
        binding.moe_decode_layer(x, wr, None, w, k, out, ws)
    for _ in range(max(3, args.warmup)):
        g_step.replay()
    torch.cuda.synchronize()
    barrier(world)

    # ---- timed region (device time, CUDA events on the launching stream)
    clocks = ClockSampler(local)
    clocks.start()
    t_beg = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    barrier(world)
    t_beg.record(stream)
    for _ in range(args.steps):
        g_step.replay()
    t_end.record(stream)
    torch.cuda.synchronize()
    ms_total = t_beg.elapsed_time(t_end)
    clk = clocks.stop()
    ms_step = barrier_max(ms_total / args.steps, world)
    tok_s = world * T / (ms_step * 1e-3)

    # per-kernel durations: eager calls with events between the kernels
    kern = [[], [], []]
    for _ in range(min(args.steps, 20)):
        step(True)
        torch.cuda.synchronize()
        for i in range(3):
            kern[i].append(ev[i].elapsed_time(ev[i + 1]))

    # ---- end to end through the public API with host buffers: the input is
    # copied from pinned host memory, the layer runs, the output is copied
    # back, every step (captured together in one graph)
    x_host = torch.empty((T, H), dtype=torch.bfloat16, pin_memory=True)
    x_host.copy_(x.cpu())
    out_host = torch.empty((T, H), dtype=torch.bfloat16, pin_memory=True)
    x_dev = torch.empty_like(x)
    g_e2e = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_e2e):
        x_dev.copy_(x_host, non_blocking=True)
        binding.moe_decode_layer(x_dev, wr, None, w, k, out, ws)
        out_host.copy_(out, non_blocking=True)
    for _ in range(3):
        g_e2e.replay()
    torch.cuda.synchronize()
    barrier(world)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        g_e2e.replay()
    e1.record(stream)
    torch.cuda.synchronize()
    ms_e2e = barrier_max(e0.elapsed_time(e1) / args.steps, world)

    # ---- energy per token (NVML counter over >= 2 s of back-to-back layers)
    energy = None
    if not args.no_energy:
        nv = Nvml(local)
        if nv.ok:
            n_rep = max(1, int(2.0 / (ms_step * 1e-3)))
            torch.cuda.synchronize()
            j0 = nv.energy_mj()
            t0 = time.perf_counter()
            for _ in range(n_rep):
                g_step.replay()
            torch.cuda.synchronize()
            dt = time.perf_counter() - t0
            j1 = nv.energy_mj()
            energy = {"j_per_token": (j1 - j0) * 1e-3 / (n_rep * T), "avg_w": (j1 - j0) * 1e-3 / dt,
                      "window_s": dt, "source": "nvmlDeviceGetTotalEnergyConsumption"}

    # ---- roofline of the dominant kernel (gate/up) and of the whole layer
    import json as _json
    peaks = {}
    pp = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(pp):
        peaks = _json.load(open(pp))
    hbm = float(peaks.get("hbm_gbs", 6800.0))
    peak_src = "measured" if "hbm_gbs" in peaks else "fallback"
    gu_ms = statistics.mean(kern[1])
    dn_ms = statistics.mean(kern[2])
    rt_ms = statistics.mean(kern[0])
    gu_alg = n_active * gu_bytes
    dn_alg = n_active * dn_bytes
    gu_gbs = gu_alg / (gu_ms * 1e-3) / 1e9
    layer_gbs = B / (ms_step * 1e-3) / 1e9
    traffic = None
    tp = os.path.join(ROOT, "profiles", "traffic.json")
    if os.path.exists(tp):
        tj = _json.load(open(tp)).get(f"{args.workload}_T{T}")
        if tj:
            traffic = tj.get("gateup_dram_bytes")

    res = {
        "metric": "MoE decode-layer tokens/s",
        "value": tok_s,
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": max(3, args.warmup),
        "ms_per_step": ms_step,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "nvfp4 weights, f16 MMA with fp32 accumulate" if fmt == 2 else
                 "fp8 weights, f16 MMA with fp32 accumulate",
        "data": "synthetic (seeded N(0,1) activations, N(0,0.02) weights quantised)",
        "config": {"workload": f"{args.workload}_T{T}", "H": H, "E": E, "k": k, "I": I,
                   "tokens": T, "format": "nvfp4" if fmt == 2 else "fp8_block128",
                   "active_experts": n_active,
                   "l2": f"inputs larger than L2: {B / 1e9:.2f} GB of weights touched per step",
                   "parallelism": f"replicas x{world}"},
        "hbm_gbs": layer_gbs,
        "hbm_frac_of_measured": layer_gbs / hbm,
        "hbm_frac_of_8tbs": layer_gbs / 8000.0,
        "algorithmic_bytes_per_step": B,
        "kernel_ms": {"route": rt_ms, "gate_up": gu_ms, "down": dn_ms},
        "roofline": {"bound": "hbm", "achieved": gu_gbs, "peak": hbm, "unit": "GB/s",
                     "frac": gu_gbs / hbm, "traffic": traffic, "kernel": "ffn gate/up",
                     "peak_source": peak_src},
        "e2e": {"value": world * T / (ms_e2e * 1e-3), "unit": "tokens/s",
                "h2d_bytes_per_step": T * H * 2, "d2h_bytes_per_step": T * H * 2},
        "gpu_launches": 5 * args.steps,
        "timing": "CUDA-graph replay of one layer call per step",
        "clocks": clk,
        "energy": energy,
    }
    if energy:
        res["j_per_token"] = energy["j_per_token"]
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        res["cpu_baseline"] = cpu_oracle_sample(fmt, H, E, k, I, T, args.seed, w=w)
    if rank == 0:
        print(json.dumps(res))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    fmt, H, E, k, I = WORKLOADS[args.workload]
    T = args.tokens
    s = OracleSample(fmt, H, E, k, I, T, args.seed, budget_s=8.0)
    warm = max(0, min(args.warmup, 1))
    for _ in range(warm):
        s.run()
    steps = max(1, min(args.steps, 5))
    dt = sum(s.run() for _ in range(steps)) / steps
    v = s.n / dt
    res = {"metric": "MoE decode-layer tokens/s", "value": v, "unit": "tokens/s", "n_gpus": world,
           "steps": steps, "warmup": warm, "ms_per_step": dt * 1e3,
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
           "data": "synthetic", "impl": "reference",
           "config": {"workload": f"{args.workload}_T{T}", "H": H, "E": E, "k": k, "I": I,
                      "tokens": T},
           "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": s.cores, "kind": "oracle",
                            "sample": f"first {s.n} of {T} tokens per step ({s.experts} experts)"},
           "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0}}
    print(json.dumps(res))


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
