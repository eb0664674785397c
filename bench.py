"""Benchmark of the MoE decode layer on GB300.

python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                [--workload NAME] [--tokens T]

One step = one decode step (router GEMV + top-k + permute + gate/up SwiGLU
+ down + combine, for each layer of the workload) over a batch of T tokens,
on synthetic seeded inputs.  Workloads:

  qwen3_480b_fp8        Qwen3-Coder-480B-shaped FP8 layer (H=6144, E=160,
                        top-8, I=2560), T=64 (the default: the largest
                        single-GPU decode layer of the two served models)
  qwen3_235b_nvfp4      Qwen3-235B-A22B-shaped NVFP4 layer (H=4096, E=128,
                        top-8, I=1536), T=64 by default
  qwen3_480b_fp8_zipf   the 480B layer with a router bias that makes expert
                        popularity follow Zipf(1.1); sweep --tokens
  qwen3_235b_nvfp4_x94  94 235B-shaped NVFP4 layers with fresh weights per
                        layer (~128 GB), RMS pre-norm and the residual stream
                        threaded between them, T=128
  qwen3_235b_nvfp4_prefill  the 235B-shaped layer on a prefill-shaped batch,
                        T=2048 (about 128 tokens per expert); its roofline is
                        the tensor-core one (useful gate/up FLOPs against the
                        dense NVFP4 peak)
  tiny_fp8              H=512, E=8, top-2, I=256, T=4

The metric is decode tokens/s; achieved HBM GB/s, the roofline fraction of
the dominant kernel (gate/up) and J/token (NVML energy counter) are reported
beside it.  The default run (N=1) adds a "sweep" key: the 235B-shaped NVFP4
layer at T = 1, 8, 32, 64, the 480B-shaped FP8 layer with Zipf-skewed
routing at T = 1, 8, 32, 128, 256 and the 235B-shaped layer on a
prefill-shaped batch of 2048 tokens (with its gate/up tensor-core fraction),
each with its time per step, layer and gate/up HBM fractions against the
measured copy rate and 8 TB/s, J/token and the SM clock over its own window
(--no-sweep skips it).  Under torchrun each rank runs an independent replica on its own
GPU (the layer does not shard across GPUs); the timed region is bracketed by
a barrier and the slowest rank's time is reported.

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
    # name: format, shape, default tokens, layers, router bias, RMS pre-norm
    "qwen3_235b_nvfp4": dict(fmt=2, H=4096, E=128, k=8, I=1536, T=64),
    "qwen3_480b_fp8": dict(fmt=1, H=6144, E=160, k=8, I=2560, T=64),
    "qwen3_480b_fp8_zipf": dict(fmt=1, H=6144, E=160, k=8, I=2560, T=64, zipf=1.1),
    "qwen3_235b_nvfp4_x94": dict(fmt=2, H=4096, E=128, k=8, I=1536, T=128, layers=94,
                                 prenorm=True),
    "qwen3_235b_nvfp4_prefill": dict(fmt=2, H=4096, E=128, k=8, I=1536, T=2048, prefill=True),
    "tiny_fp8": dict(fmt=1, H=512, E=8, k=2, I=256, T=4),
}
MOE_FLAG_PRENORM_RMS = 0x2
MOE_FLAG_DETERMINISTIC = 0x4


def workload(args):
    wl = dict(layers=1, zipf=None, prenorm=False, prefill=False)
    wl.update(WORKLOADS[args.workload])
    if args.tokens is not None:
        wl["T"] = args.tokens
    if args.experts is not None:
        wl["E"] = args.experts
    wl["det"] = bool(getattr(args, "deterministic", False))
    wl["name"] = args.workload + (f"_E{wl['E']}" if args.experts is not None else "") \
        + f"_T{wl['T']}" + ("_det" if wl["det"] else "")
    return wl


def parse(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="qwen3_480b_fp8", choices=sorted(WORKLOADS))
    ap.add_argument("--tokens", type=int, default=None, help="batch size (default per workload)")
    ap.add_argument("--experts", type=int, default=None,
                    help="expert count (default per workload); a smaller count keeps the "
                         "layer's per-expert shapes with less memory, for profiler captures")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-energy", action="store_true")
    ap.add_argument("--no-sweep", action="store_true",
                    help="skip the batch sweep of the default run")
    ap.add_argument("--deterministic", action="store_true",
                    help="run the layer with MOE_FLAG_DETERMINISTIC (the same output bits "
                         "on every run)")
    return ap.parse_args(argv)


# ---------------------------------------------------------------- distributed
def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def barrier_max(value, world):
    """Barrier, then the maximum of `value` over ranks (an all-reduce, so every
    rank returns the slowest rank's figure).  The reduction buffer lives where
    the process group's backend wants it: the GPU for nccl, the host for gloo."""
    if world == 1:
        return value
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([value], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(ms_step_max, tokens_per_rank, world):
    """Whole-job tokens/s of `world` replicas, each decoding `tokens_per_rank`
    tokens per step, paced by the slowest rank's step time."""
    return world * tokens_per_rank / (ms_step_max * 1e-3)


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


# ---------------------------------------------------------------- clocks / energy
class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons, each stamped with
    the host time it arrived, so that a window of them can be kept."""

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
            self.lines.append((time.perf_counter(), line.strip()))

    def running(self):
        return self.proc is not None and self.proc.poll() is None

    def stop(self, t0=None, t1=None):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        return self.summary(t0, t1)

    def summary(self, t0=None, t1=None):
        """Median SM clock, max clock, throttle reasons and median power of the
        samples that arrived between host times t0 and t1."""
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        sm, smax, reasons, watts = [], None, set(), []
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ts, ln in list(self.lines):
            if (t0 is not None and ts < t0) or (t1 is not None and ts > t1):
                continue
            f = [v.strip() for v in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax = float(f[2])
                watts.append(float(f[3]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": smax,
                "reasons": sorted(reasons), "samples": len(sm),
                "power_w_median": statistics.median(watts) if watts else None}


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


# ---------------------------------------------------------------- synthetic workload
def layer_seed(seed, layer):
    """Seed of layer `layer`'s weights and router (fresh weights per layer)."""
    return seed + 1009 * layer


def zipf_bias(wl, seed, device):
    from paper_2609_11133_gb300 import synth
    if not wl["zipf"]:
        return None
    return synth.make_zipf_bias(wl["E"], wl["H"], s=wl["zipf"], seed=seed, device=device)


# ---------------------------------------------------------------- CPU oracle
def _oracle_weights(w, experts=None):
    """The oracle's copy of w; with `experts`, only those experts are copied
    (the others stay zero; numpy's zeros are not touched until written)."""
    import numpy as np

    from oracle import oracle
    ts = (w.w_gate, w.w_up, w.w_down, w.s_gate, w.s_up, w.s_down, w.ts_gate, w.ts_up, w.ts_down)
    if experts is None:
        return oracle.ExpertWeights(w.fmt, w.E, w.H, w.I, *[
            None if t is None else t.detach().cpu().numpy() for t in ts])
    out = []
    for t in ts:
        if t is None:
            out.append(None)
            continue
        a = np.zeros(tuple(t.shape), dtype=t.cpu()[:0].numpy().dtype)
        for e in experts:
            a[int(e)] = t[int(e)].detach().cpu().numpy()
        out.append(a)
    return oracle.ExpertWeights(w.fmt, w.E, w.H, w.I, *out)


class OracleSample:
    """The float64 oracle (RMS pre-norm if the workload has it, router, top-k,
    experts, combine) on the first n tokens of layer 0 of the workload, on the
    host cores.  n is chosen so that one pass takes about `budget_s` seconds;
    only the experts those tokens route to are generated (on the host,
    untimed) unless the full weights are given."""

    def __init__(self, wl, seed, budget_s=10.0, w=None):
        import numpy as np
        import torch

        from oracle import oracle
        from paper_2609_11133_gb300 import synth
        fmt, H, E, k, I, T = (wl[n] for n in ("fmt", "H", "E", "k", "I", "T"))
        self.k = k
        self.prenorm = wl["prenorm"]
        self.cores = len(os.sched_getaffinity(0))
        x = synth.make_x(T, H, seed=seed)
        self.xb = x.view(torch.int16).numpy().view(np.uint16)
        s0 = layer_seed(seed, 0)
        self.wr = synth.make_router(E, H, seed=s0).numpy()
        b = zipf_bias(wl, seed, "cpu")
        self.bias = None if b is None else b.numpy()
        xr = oracle.rmsnorm_bf16(self.xb) if self.prenorm else self.xb
        ids, _ = oracle.topk(oracle.router_logits(xr, self.wr, self.bias), k)
        # calibrate on one token; weights given (the device's): copy only the
        # experts the sample routes to; else generate only those on the host
        def weights_for(n_tok):
            ex = np.unique(ids[:n_tok])
            if w is not None:
                return _oracle_weights(w, ex)
            return _oracle_weights(synth.make_weights(fmt, E, H, I, seed=s0, experts=ex))
        self.ow = weights_for(1)
        self.n = 1
        dt = self.run()
        n = max(1, min(T, int(budget_s / max(dt, 1e-3))))
        self.n = n
        if n > 1:
            self.ow = weights_for(n)
        self.experts = int(np.unique(ids[:n]).size)

    def run(self):
        from oracle import oracle
        sub = self.xb[:self.n]
        t0 = time.perf_counter()
        xr = oracle.rmsnorm_bf16(sub) if self.prenorm else sub
        ids, gates = oracle.topk(oracle.router_logits(xr, self.wr, self.bias), self.k)
        oracle.moe_tokens(self.ow, xr, ids, gates, residual_bits=sub if self.prenorm else None)
        return time.perf_counter() - t0


def _omp_threads(n=None):
    """The OpenMP thread count of this process (the oracle's), set if n is given."""
    try:
        gomp = ctypes.CDLL("libgomp.so.1")
    except OSError:
        return None
    if n is not None:
        gomp.omp_set_num_threads(int(n))
    return gomp.omp_get_max_threads()


def cpu_oracle_sample(wl, seed, w=None, budget_s=10.0):
    s = OracleSample(wl, seed, budget_s=budget_s, w=w)
    dt = s.run()
    L = wl["layers"]
    per_layer = f", x{L} layers (layer 0 timed)" if L > 1 else ""
    res = {"value": s.n / (dt * L), "unit": "tokens/s", "cores": s.cores, "kind": "oracle",
           "sample": f"first {s.n} of {wl['T']} tokens ({s.experts} experts): "
                     f"{'RMS pre-norm, ' if wl['prenorm'] else ''}router, top-k, experts and "
                     f"combine in float64, {dt:.2f} s{per_layer}"}
    # the same oracle on one core, on the first token of the sample
    prev = _omp_threads()
    if prev:
        n_all = s.n
        try:
            _omp_threads(1)
            s.n = 1
            dt1 = s.run()
        finally:
            s.n = n_all
            _omp_threads(prev)
        res["one_core"] = {"value": 1.0 / (dt1 * L), "unit": "tokens/s",
                           "sample": f"first token, {dt1:.2f} s{per_layer}"}
    return res


def expert_bytes(w):
    """(gate+up, down) stored bytes of one expert: codes + scales."""
    gu = (w.w_gate[0].numel() + w.w_up[0].numel()) + \
        (w.s_gate[0].numel() * w.s_gate.element_size() + w.s_up[0].numel() * w.s_up.element_size())
    dn = w.w_down[0].numel() + w.s_down[0].numel() * w.s_down.element_size()
    if w.fmt == 2:
        gu += 8
        dn += 4
    return gu, dn


def zipf_stats(ids, E):
    """Realised expert popularity of a routed batch: counts, and the exponent
    of a least-squares fit log n_e = c - s log rank over the experts used."""
    import numpy as np
    cnt = np.bincount(ids.reshape(-1), minlength=E)
    srt = np.sort(cnt)[::-1]
    nz = srt[srt > 0]
    fit = None
    if nz.size >= 3:
        r = np.log(np.arange(1, nz.size + 1))
        fit = float(-np.polyfit(r, np.log(nz), 1)[0])
    return {"max_n_e": int(srt[0]), "top5_n_e": [int(v) for v in srt[:5]],
            "fitted_s": fit}


def kernel_sources_sha256():
    """sha256 over every CUDA source of the library (sorted by name)."""
    import hashlib
    d = os.path.join(ROOT, "paper_2609_11133_gb300", "csrc")
    h = hashlib.sha256()
    for f in sorted(os.listdir(d)):
        if f.endswith((".cu", ".cuh")):
            h.update(f.encode())
            h.update(open(os.path.join(d, f), "rb").read())
    return h.hexdigest()


# ---------------------------------------------------------------- our arm
def metric_name(wl):
    """The metric both arms report for a workload."""
    if wl["layers"] > 1:
        return f"MoE {wl['layers']}-layer decode-step tokens/s"
    return "MoE prefill-shaped layer tokens/s" if wl["prefill"] else "MoE decode-layer tokens/s"


def gateup_roofline(wl, fmt, T, k, H, I, gu_ms, gu_gbs, peaks, traffic):
    """The `roofline` object of the dominant kernel, gate/up.  Decode batches:
    algorithmic bytes per launch / its CUDA-event time against the measured
    copy rate.  A prefill-shaped batch reuses each weight tile for ~T*k/E
    tokens, so its roofline is the tensor cores': useful gate/up FLOPs (2
    matrices x 2 x H x I per assignment; the activation terms' extra MMA work
    is not counted) against the dense rate of the weights' format, the
    measured sustained bf16 rate times the nominal ratio (NVFP4 13.5 / 2.25 =
    6, FP8 4.5 / 2.25 = 2)."""
    hbm = float(peaks.get("hbm_gbs", 6800.0))
    hbm_src = "measured" if "hbm_gbs" in peaks else "fallback"
    if not wl["prefill"]:
        return {"bound": "hbm", "achieved": gu_gbs, "peak": hbm, "unit": "GB/s",
                "frac": gu_gbs / hbm, "traffic": traffic, "kernel": "ffn gate/up",
                "peak_source": hbm_src}
    ratio, name = (6.0, "NVFP4") if fmt == 2 else (2.0, "FP8")
    tflops = 4.0 * T * k * H * I / (gu_ms * 1e-3) / 1e12
    bf16 = peaks.get("bf16_tflops_sustained")
    peak = ratio * (float(bf16) if bf16 else 1700.0)
    src = (f"measured bf16 sustained x {ratio:g} ({name})" if bf16 else
           f"fallback 1.7 PFLOP/s bf16 sustained x {ratio:g} ({name})")
    return {"bound": "tensor", "achieved": tflops, "peak": peak, "unit": "TFLOP/s",
            "frac": tflops / peak, "traffic": traffic, "kernel": "ffn gate/up",
            "peak_source": src,
            "hbm": {"achieved": gu_gbs, "peak": hbm, "unit": "GB/s", "frac": gu_gbs / hbm}}


class Runner:
    """One workload at one batch size on this GPU: the layers' weights, the
    resident input batches, a workspace, and the timings of this file.

    Steps rotate over distinct input batches, all resident before timing, when
    one step touches less than four times L2: consecutive steps then route to
    different experts and a step does not find the weights of the previous ones
    in L2.  Steps are replayed from CUDA graphs of G steps (one rotation cycle,
    at least eight layer calls); within a graph the layer calls follow one
    another as in a decode loop and the host takes no decision between them."""

    def __init__(self, wl, layers, bias, seed, rank, dev="cuda"):
        import torch

        from paper_2609_11133_gb300 import binding, synth
        self.torch, self.binding = torch, binding
        self.wl, self.layers, self.bias = wl, layers, bias
        self.T, self.H, self.k, self.E, self.L = wl["T"], wl["H"], wl["k"], wl["E"], wl["layers"]
        self.flags = (MOE_FLAG_PRENORM_RMS if wl["prenorm"] else 0) | \
            (MOE_FLAG_DETERMINISTIC if wl.get("det") else 0)
        T, H = self.T, self.H
        self.dev = dev
        x = synth.make_x(T, H, seed=seed + rank, device=dev)
        # the residual stream of a stack: layer l reads cur and writes nxt
        self.bufs = [torch.empty((T, H), dtype=torch.bfloat16, device=dev) for _ in range(2)]
        self.ws = binding.alloc_workspace(
            binding.moe_workspace_size(layers[0][0], T, self.k, self.flags))
        self.stream = torch.cuda.current_stream()
        w0 = layers[0][0]
        self.gu_bytes, self.dn_bytes = expert_bytes(w0)
        self.per_expert = w0.nbytes_expert()
        self.router_bytes = self.E * H * 4
        self.act_bytes = 2 * T * H * 2  # x in, out
        n_active, self.ids, B = self.touched(x)
        l2 = torch.cuda.get_device_properties(0).L2_cache_size
        self.l2 = l2
        self.n_rot = 1 if B >= 4 * l2 else min(16, math.ceil(4 * l2 / B))
        self.xs = [x] + [synth.make_x(T, H, seed=seed + rank + 7919 * r, device=dev)
                         for r in range(1, self.n_rot)]
        if self.n_rot > 1:
            rot = [self.touched(xr) for xr in self.xs]
            n_active = [statistics.mean(r[0][l] for r in rot) for l in range(self.L)]
            B = statistics.mean(r[2] for r in rot)
        self.n_active, self.B = n_active, B
        self.G = self.n_rot * max(1, math.ceil(8 / (self.n_rot * self.L)))

    def io(self, l, x_in):
        """(input, residual, output) of layer l."""
        if self.L == 1:
            return x_in, None, self.bufs[0]
        cur = x_in if l == 0 else self.bufs[(l - 1) % 2]
        return cur, cur, self.bufs[l % 2]

    def run_layers(self, x_in, ev=None, ids=None):
        b = self.binding
        for l, (w, wr) in enumerate(self.layers):
            xi, res, out = self.io(l, x_in)
            if ev is None and ids is None:
                b.moe_decode_layer(xi, wr, self.bias, w, self.k, out, self.ws, flags=self.flags,
                                   residual=res)
            else:
                b.moe_decode_layer_ex(xi, wr, self.bias, w, self.k, out, self.ws,
                                      flags=self.flags, residual=res,
                                      events=None if ev is None else ev[l],
                                      topk_ids_out=None if ids is None else ids[l])
        return self.io(self.L - 1, x_in)[2]

    def touched(self, x_in):
        """Unique experts per layer of one batch, and the step's algorithmic bytes."""
        torch = self.torch
        ids = [torch.empty((self.T, self.k), dtype=torch.int32, device=self.dev)
               for _ in range(self.L)]
        self.run_layers(x_in, ids=ids)
        torch.cuda.synchronize()
        assert self.binding.moe_read_status(self.ws) == 0
        n = [int(torch.unique(i).numel()) for i in ids]
        return n, ids, sum(self.router_bytes + a * self.per_expert + self.act_bytes for a in n)

    def capture(self, nsteps, body):
        g = self.torch.cuda.CUDAGraph()
        with self.torch.cuda.graph(g):
            for s_ in range(nsteps):
                body(s_ % self.n_rot)
        return g

    def graphs(self, steps, body=None):
        body = body or (lambda r: self.run_layers(self.xs[r]))
        g_full = self.capture(self.G, body)
        g_rem = self.capture(steps % self.G, body) if steps % self.G else None
        return g_full, g_rem

    def timed(self, g_full, g_rem, steps, marks=None):
        """Replays that run exactly `steps` steps; `marks` gets an event after
        every full replay (the spread over repetitions)."""
        for _ in range(steps // self.G):
            g_full.replay()
            if marks is not None:
                marks.append(self.torch.cuda.Event(enable_timing=True))
                marks[-1].record(self.stream)
        if g_rem is not None:
            g_rem.replay()

    def warm(self, g_full, warmup):
        for _ in range(max(3, warmup)):
            self.run_layers(self.xs[0])
        for _ in range(max(3, math.ceil(warmup / self.G))):
            g_full.replay()
        self.torch.cuda.synchronize()

    def time_steps(self, g_full, g_rem, steps, world, marks=None):
        """Device time of exactly `steps` steps (ms per step, max over ranks),
        bracketed by a barrier and a synchronisation on both sides; host
        times of the region."""
        torch = self.torch
        t_beg = torch.cuda.Event(enable_timing=True)
        t_end = torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        barrier(world)
        h_beg = time.perf_counter()
        t_beg.record(self.stream)
        self.timed(g_full, g_rem, steps, marks)
        t_end.record(self.stream)
        torch.cuda.synchronize()
        h_end = time.perf_counter()
        ms = t_beg.elapsed_time(t_end)
        reps = None
        if marks:
            reps = [a.elapsed_time(b) / self.G for a, b in zip([t_beg] + marks[:-1], marks)]
        return barrier_max(ms / steps, world), h_beg, h_end, reps

    def energy(self, g_full, ms_step, local, seconds):
        """J/token from the NVML energy counter over >= `seconds` of
        back-to-back steps; (result, host end time)."""
        torch = self.torch
        nv = Nvml(local)
        if not nv.ok:
            return None, time.perf_counter()
        n_rep = max(1, int(seconds / (ms_step * 1e-3 * self.G)))
        torch.cuda.synchronize()
        j0 = nv.energy_mj()
        t0 = time.perf_counter()
        for _ in range(n_rep):
            g_full.replay()
        torch.cuda.synchronize()
        t1 = time.perf_counter()
        j1 = nv.energy_mj()
        return {"j_per_token": (j1 - j0) * 1e-3 / (n_rep * self.G * self.T),
                "avg_w": (j1 - j0) * 1e-3 / (t1 - t0), "window_s": t1 - t0,
                "source": "nvmlDeviceGetTotalEnergyConsumption"}, t1

    def kernel_ms(self, n):
        """Mean CUDA-event durations (ms per layer) of route (+ gather), gate/up
        and SwiGLU + down + finalize, from eager calls with events between
        the kernels on the launching stream."""
        torch = self.torch
        ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(self.L)]
        kern = [[], [], []]
        for i_ in range(n):
            self.run_layers(self.xs[i_ % self.n_rot], ev=ev)
            torch.cuda.synchronize()
            for i in range(3):
                kern[i].append(sum(ev[l][i].elapsed_time(ev[l][i + 1]) for l in range(self.L)))
        return [statistics.mean(k_) / self.L for k_ in kern]

    def hbm(self, ms_step, gu_ms, peaks):
        hbm = float(peaks.get("hbm_gbs", 6800.0))
        gu_alg = statistics.mean(self.n_active) * self.gu_bytes  # per launch
        gu_gbs = gu_alg / (gu_ms * 1e-3) / 1e9
        layer_gbs = self.B / (ms_step * 1e-3) / 1e9
        return {"layer_gbs": layer_gbs, "layer_frac_of_measured": layer_gbs / hbm,
                "layer_frac_of_8tbs": layer_gbs / 8000.0, "gateup_gbs": gu_gbs,
                "gateup_frac_of_measured": gu_gbs / hbm, "gateup_frac_of_8tbs": gu_gbs / 8000.0}


def load_peaks():
    pp = os.path.join(ROOT, "MEASURED_PEAKS.json")
    return json.load(open(pp)) if os.path.exists(pp) else {}


def make_layers(wl, seed, dev="cuda"):
    from paper_2609_11133_gb300 import synth
    out = []
    for l in range(wl["layers"]):
        sl = layer_seed(seed, l)
        out.append((synth.make_weights(wl["fmt"], wl["E"], wl["H"], wl["I"], seed=sl, device=dev),
                    synth.make_router(wl["E"], wl["H"], seed=sl, device=dev)))
    return out


# The sweep of the default run: (workload, batch sizes).  The 480B-shaped
# layers reuse the headline's weights (same seed); only the router bias and
# the batch differ.
SWEEP = [("qwen3_235b_nvfp4", (1, 8, 32, 64)), ("qwen3_480b_fp8_zipf", (1, 8, 32, 128, 256)),
         ("qwen3_235b_nvfp4_prefill", (2048,))]
SWEEP_TIMED_S = 0.25   # timed device work per sweep entry
SWEEP_ENERGY_S = 1.0   # energy window per sweep entry


def sweep_entry(run, peaks, clocks, local, no_energy):
    """Time, HBM fractions, J/token and clocks of one sweep entry."""
    g_full, _ = run.graphs(0)
    run.warm(g_full, 3)
    ms0, _, _, _ = run.time_steps(g_full, None, run.G, 1)
    steps = max(50, run.G * math.ceil(SWEEP_TIMED_S / (ms0 * 1e-3) / run.G))
    ms, h0, h1, _ = run.time_steps(g_full, None, steps, 1)
    energy = None
    if not no_energy:
        energy, h1 = run.energy(g_full, ms, local, SWEEP_ENERGY_S)
    rt, gu, dn = run.kernel_ms(20)
    clk = clocks.summary(h0, h1)
    e = {"tokens": run.T, "ms_per_step": ms, "tokens_per_s": run.T / (ms * 1e-3),
         "steps": steps, "active_experts": statistics.mean(run.n_active),
         "algorithmic_bytes_per_step": run.B,
         "kernel_ms": {"route": rt, "gate_up": gu, "down": dn}}
    e.update(run.hbm(ms, gu, peaks))
    if run.wl["prefill"]:  # the tensor-core roofline of the gate/up kernel
        wl = run.wl
        rf = gateup_roofline(wl, wl["fmt"], run.T, run.k, run.H, wl["I"], gu,
                             e["gateup_gbs"], peaks, None)
        e["gateup_tensor"] = {k_: rf[k_] for k_ in ("achieved", "peak", "unit", "frac",
                                                    "peak_source")}
    e["j_per_token"] = energy["j_per_token"] if energy else None
    e["sm_mhz_median"] = clk.get("sm_mhz")
    e["clock_reasons"] = clk.get("reasons")
    if run.wl["zipf"]:
        e["popularity"] = zipf_stats(run.ids[0].cpu().numpy(), run.E)
    return e


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
    from paper_2609_11133_gb300 import binding

    wl = workload(args)
    fmt, H, E, k, I, T, L = (wl[n] for n in ("fmt", "H", "E", "k", "I", "T", "layers"))
    dev = "cuda"
    layers = make_layers(wl, args.seed, dev)
    run = Runner(wl, layers, zipf_bias(wl, args.seed, dev), args.seed, rank, dev)
    G, n_rot = run.G, run.n_rot

    g_step, g_rem = run.graphs(args.steps)
    run.warm(g_step, args.warmup)
    barrier(world)

    # clock sampler: started before the timed region; the replays below keep
    # the GPU busy until its first sample arrives (bounded), so that the
    # samples kept cover the timed region and the energy window only
    clocks = ClockSampler(local)
    clocks.start()
    t_wait = time.perf_counter()
    while clocks.running() and not clocks.lines and time.perf_counter() - t_wait < 5.0:
        g_step.replay()
        torch.cuda.synchronize()

    # ---- timed region (device time, CUDA events on the launching stream)
    marks = []
    ms_step, h_beg, h_end, reps = run.time_steps(g_step, g_rem, args.steps, world, marks)
    tok_s = job_throughput(ms_step, T, world)
    repeats = None
    if reps:
        repeats = {"n": len(reps), "steps_each": G, "median_ms": float(np.median(reps)),
                   "p10_ms": float(np.percentile(reps, 10)),
                   "p90_ms": float(np.percentile(reps, 90))}

    # ---- energy per token (NVML counter over >= 2 s of back-to-back steps)
    energy = None
    if not args.no_energy:
        energy, h_end = run.energy(g_step, ms_step, local, 2.0)
    clk = clocks.summary(h_beg, h_end)
    clk["window"] = "timed region" + (" + energy window (same steps replayed)" if energy else "")

    # single-call latency: one step, eager (host launches included) and as a
    # one-step graph, each timed alone on an idle GPU
    lat_eager, lat_graph = [], []
    g_one = run.capture(1, lambda r: run.run_layers(run.xs[r]))
    for i_ in range(12):
        a_, b_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        a_.record(run.stream)
        if i_ % 2:
            g_one.replay()
        else:
            run.run_layers(run.xs[0])
        b_.record(run.stream)
        torch.cuda.synchronize()
        (lat_graph if i_ % 2 else lat_eager).append(a_.elapsed_time(b_) * 1e3)
    latency = {"eager_us": statistics.median(lat_eager[1:]),
               "graph_us": statistics.median(lat_graph[1:]),
               "per": "layer call" if L == 1 else f"{L}-layer step"}

    # per-kernel durations: eager calls with events between the kernels
    rt_ms, gu_ms, dn_ms = run.kernel_ms(max(1, min(args.steps, 20 if L == 1 else 2)))

    # ---- end to end through the public API with host buffers: every step
    # copies its input from pinned host memory, runs, and copies its output
    # back (the same steps per graph and the same input rotation)
    x_host = [torch.empty((T, H), dtype=torch.bfloat16, pin_memory=True) for _ in range(n_rot)]
    for xh, xr in zip(x_host, run.xs):
        xh.copy_(xr.cpu())
    out_host = torch.empty((T, H), dtype=torch.bfloat16, pin_memory=True)
    x_dev = torch.empty_like(run.xs[0])

    def e2e_step(r):
        x_dev.copy_(x_host[r], non_blocking=True)
        o = run.run_layers(x_dev)
        out_host.copy_(o, non_blocking=True)

    g_e2e, g_e2e_rem = run.graphs(args.steps, e2e_step)
    for _ in range(3):
        g_e2e.replay()
    torch.cuda.synchronize()
    ms_e2e, _, _, _ = run.time_steps(g_e2e, g_e2e_rem, args.steps, world)
    assert torch.isfinite(out_host.float()).all()

    # ---- roofline of the dominant kernel (gate/up) and of the whole step
    peaks = load_peaks()
    hb = run.hbm(ms_step, gu_ms, peaks)
    # DRAM bytes of one gate/up launch from a committed ncu capture, valid only
    # while the kernel sources are the ones that capture was taken on
    traffic = None
    tp = os.path.join(ROOT, "profiles", "traffic.json")
    if os.path.exists(tp):
        tj = json.load(open(tp)).get(wl["name"])
        if tj and kernel_sources_sha256() == tj.get("kernel_sources_sha256"):
            traffic = tj.get("gateup_dram_bytes")

    B = run.B
    cfg = {"workload": wl["name"], "H": H, "E": E, "k": k, "I": I,
           "tokens": T, "format": "nvfp4" if fmt == 2 else "fp8_block128",
           "active_experts": run.n_active[0] if L == 1 else statistics.mean(run.n_active),
           "l2": (f"inputs larger than L2: {B / 1e9:.2f} GB of weights touched per step"
                  if n_rot == 1 else
                  f"{n_rot} resident input batches rotated step by step: {B / 1e9:.3f} GB "
                  f"touched per step, {n_rot * B / 1e9:.2f} GB per rotation "
                  f"(L2 {run.l2 / 1e6:.0f} MB)"),
           "steps_per_graph": G,
           "arithmetic": ("e2m1 x e2m1 block-scaled MMA (ue4m3 per 16), activations as 4 nvfp4 "
                          "terms, fp32 accumulate" if fmt == 2 else
                          "e4m3 x e4m3 MMA, 128x128 fp32 block scales applied per stage, "
                          "activations as 2 e4m3 terms, fp32 accumulate"),
           "parallelism": f"replicas x{world}"}
    if wl["det"]:
        cfg["deterministic"] = "MOE_FLAG_DETERMINISTIC (down step timed with its combine)"
    if L > 1:
        cfg.update(layers=L, prenorm="rms, eps 1e-6, unit weight", residual="threaded",
                   weights_gb=round(sum(w.nbytes_expert() * E for w, _ in layers) / 1e9, 1))
    if wl["zipf"]:
        cfg["router_bias"] = f"zipf s={wl['zipf']}"
        cfg["popularity"] = zipf_stats(run.ids[0].cpu().numpy(), E)
    roofline = gateup_roofline(wl, fmt, T, k, H, I, gu_ms, hb["gateup_gbs"], peaks, traffic)
    res = {
        "metric": metric_name(wl),
        "value": tok_s,
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": max(3, args.warmup),
        "ms_per_step": ms_step,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "nvfp4" if fmt == 2 else "fp8_e4m3",
        "data": "synthetic (seeded N(0,1) activations, N(0,0.02) weights quantised)",
        "config": cfg,
        "hbm_gbs": hb["layer_gbs"],
        "hbm_frac_of_measured": hb["layer_frac_of_measured"],
        "hbm_frac_of_8tbs": hb["layer_frac_of_8tbs"],
        "gateup_frac_of_8tbs": hb["gateup_frac_of_8tbs"],
        "algorithmic_bytes_per_step": B,
        "kernel_ms": {"route": rt_ms, "gate_up": gu_ms, "down": dn_ms,
                      "per": "layer" if L == 1 else f"layer, mean of {L}"},
        "roofline": roofline,
        "e2e": {"value": job_throughput(ms_e2e, T, world), "unit": "tokens/s",
                "h2d_bytes_per_step": T * H * 2, "d2h_bytes_per_step": T * H * 2},
        "gpu_launches": binding.moe_layer_kernel_count(layers[0][0], T, k) * L * args.steps,
        "timing": f"CUDA-graph replay, {G} steps (layer calls) per graph",
        "repeats": repeats,
        "latency": latency,
        "clocks": clk,
        "energy": energy,
    }
    if energy:
        res["j_per_token"] = energy["j_per_token"]

    # ---- the batch sweep (default run, one GPU): other batch sizes and the
    # other served model's layer, each measured over its own window
    if world == 1 and not args.no_sweep and args.workload == "qwen3_480b_fp8" \
            and args.tokens is None and args.experts is None:
        sweep = {}
        for name, batches in SWEEP:
            base = dict(layers=1, zipf=None, prenorm=False, prefill=False)
            base.update(WORKLOADS[name])
            lay = layers if base["fmt"] == fmt and base["E"] == E and base["H"] == H \
                and base["I"] == I else make_layers(base, args.seed, dev)
            bias = zipf_bias(base, args.seed, dev)
            for t_ in batches:
                wl_t = dict(base, T=t_, name=f"{name}_T{t_}")
                r_t = Runner(wl_t, lay, bias, args.seed, rank, dev)
                sweep[wl_t["name"]] = sweep_entry(r_t, peaks, clocks, local, args.no_energy)
                del r_t
            if lay is not layers:
                del lay
                torch.cuda.empty_cache()
        res["sweep"] = sweep
    clocks.stop()

    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        res["cpu_baseline"] = cpu_oracle_sample(wl, args.seed, w=layers[0][0])  # layer 0
    if rank == 0:
        print(json.dumps(res))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    wl = workload(args)
    T, L = wl["T"], wl["layers"]
    steps, warm = max(1, args.steps), max(0, args.warmup)
    # each step is a bounded token sample, sized so the whole run takes ~2 min
    budget = min(8.0, max(0.3, 120.0 / (steps + warm)))
    s = OracleSample(wl, args.seed, budget_s=budget)
    for _ in range(warm):
        s.run()
    dt = sum(s.run() for _ in range(steps)) / steps
    v = s.n / (dt * L)
    res = {"metric": metric_name(wl),
           "value": v, "unit": "tokens/s", "n_gpus": world,
           "steps": steps, "warmup": warm, "ms_per_step": dt * L * 1e3,
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
           "data": "synthetic", "impl": "reference",
           "config": {"workload": wl["name"], "H": wl["H"], "E": wl["E"],
                      "k": wl["k"], "I": wl["I"], "tokens": T,
                      "step": f"the first {s.n} of the batch's {T} tokens (a bounded sample); "
                              f"ms_per_step is the time of that sample"
                              + (f", layer 0 timed and counted {L} times" if L > 1 else "")},
           "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": s.cores, "kind": "oracle",
                            "sample": f"first {s.n} of {T} tokens per step ({s.experts} experts)"
                                      + (f", layer 0 of {L}" if L > 1 else "")},
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
