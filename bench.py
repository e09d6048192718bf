"""Benchmark of the MomentKV hot path on GB300.

A step is one pass of the whole path over one synthetic layer of the
Llama-3.1-8B attention geometry (32 query heads, 8 KV heads, d=128, bf16,
batch 1): compress a T=8192 prompt to a budget of 512 (window 32, one sink,
moment filter on), then 256 corrected decode steps, each appending its token,
with a moment-informed eviction back to the budget after every 64 tokens.
Each part is captured once in a CUDA graph and replayed; CUDA events on the
launching stream time the segments.  L2 is flushed (a 256 MB write) before
every timed step, outside the timed region.

value      generated decode tokens per second of whole-step time (device-timed,
           inputs resident in HBM).
e2e        the same with the step's inputs copied from pinned host memory and
           the decode outputs copied back inside the timed region.
roofline   the dominant kernel against the measured HBM copy bandwidth.
extra keys the decode sweep cells (batch x budget, correction on/off),
           compress throughput at 32K and 128K context, the continuous
           eviction mode (one Algorithm 1 step per token at the budget), and
           32 layers' decode in one launch against one launch per layer.

--impl reference times the fp64 oracle on the host cores instead (a bounded
sample: one KV-head unit of the same workload per step, scaled to the whole).
--only LEG runs one of the extra legs alone and prints its result, so that a
profiler can capture that leg without the step's decode launches.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import resource
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "decode-step attn+correction tokens/s and HBM GB/s frac; compress GB/s at 1 GB300"
WORKLOAD = "llama8b_layer_t8k"
EVICT_EVERY = 64

# dram__bytes_read.sum + dram__bytes_write.sum per launch of the dominant
# kernel from one ncu capture of the bench workload
# (profiles/decode_kernel_llama8b_layer_t8k.md), valid while the code the
# kernel compiles from (its .cu file and the library headers, comments
# aside) is what was captured: code_sha of those sources at capture time.
NCU_TRAFFIC = {"decode": {"bytes": 2957824,
                          "code_sha": "91f03de032396f51c39e95e171ace5ef6b207ef5a5e4cec27397692c8a88dba9"}}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--no-extras", action="store_true", help="skip the decode sweep and long-context compress")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--only", choices=["decode_sweep", "compress_long", "continuous_eviction", "layers_one_launch"],
                    help="run one extra leg alone and print its result (for profiling that leg)")
    return ap.parse_args()


def job_throughput(total_ms, steps, tokens_per_rank, dist=None, device=None):
    """Whole-job timing of `steps` timed steps over the ranks (one replica per
    GPU): the slowest rank's total time, and the tokens all ranks processed in
    it.  Returns (ms per step, tokens/s)."""
    world = 1
    if dist is not None:
        import torch
        t = torch.tensor([total_ms], dtype=torch.float64, device=device)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        total_ms = float(t.item())
        world = dist.get_world_size()
    ms_per_step = total_ms / steps
    return ms_per_step, tokens_per_rank * world / (ms_per_step / 1e3)


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def kernel_sources(cu):
    """The files a kernel compiles from: its .cu file and the library headers."""
    c = os.path.join(ROOT, "paper_2606_01563_gb300", "csrc")
    return [os.path.join(c, cu), os.path.join(c, "common.cuh"), os.path.join(c, "kernels.h"),
            os.path.join(ROOT, "include", "mkv.h")]


def code_sha(paths):
    """sha256 of C/CUDA sources' code alone (the files in order): comments
    removed and every run of whitespace collapsed to one space, string and
    character literals kept as written.  An edit to comments leaves it
    unchanged; any edit to the code changes it."""
    src = ""
    for path in paths:
        with open(path) as f:
            src += f.read() + "\n"
    out, i, n = [], 0, len(src)
    while i < n:
        c = src[i]
        if src.startswith("//", i):
            j = src.find("\n", i)
            i = n if j < 0 else j
            out.append(" ")
        elif src.startswith("/*", i):
            j = src.find("*/", i + 2)
            i = n if j < 0 else j + 2
            out.append(" ")
        elif c in "\"'":
            j = i + 1
            while j < n and src[j] != c:
                j += 2 if src[j] == "\\" else 1
            out.append(src[i:j + 1])
            i = j + 1
        else:
            out.append(c)
            i += 1
    code = " ".join("".join(out).split())
    return hashlib.sha256(code.encode()).hexdigest()


# --------------------------------------------------------------------------
# clocks during the timed region
# --------------------------------------------------------------------------
class Clocks:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index):
        self.proc = None
        self.idx = device_index

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out = ""
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 7:
                continue
            try:
                sm.append(float(f[0]))
                mx.append(float(f[1]))
            except ValueError:
                continue
            for n, v in zip(names, f[3:7]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": float(np.median(sm)) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "samples": len(sm), "reasons": sorted(reasons)}


# --------------------------------------------------------------------------
# the GPU step
# --------------------------------------------------------------------------
class Step:
    """Device state, CUDA graphs and byte counts for one workload replica."""

    def __init__(self, torch, mkv, inputs, seed, dev):
        self.t = torch
        self.mkv = mkv
        wl = inputs.WORKLOADS[WORKLOAD]
        self.wl = wl
        G = wl.geom
        self.G = G
        self.g = mkv.geom(G.batch, G.n_kv_heads, G.group, G.head_dim)
        self.dev = dev
        gen = inputs.Generator(wl, seed=seed)
        K, V, Q = gen.prefill()
        q, kn, vn = gen.decode(wl.decode_steps)
        tb = inputs.to_bf16_tensor
        # pinned host copies (e2e) and device copies (value)
        self.host_in = {k: tb(x).pin_memory() for k, x in (("K", K), ("V", V), ("Q", Q), ("q", q), ("kn", kn),
                                                          ("vn", vn))}
        self.dev_in = {k: v.to(dev) for k, v in self.host_in.items()}
        self.T, self.B, self.S = wl.T, wl.budget, wl.decode_steps
        self.cap = self.B + EVICT_EVERY
        self.p = mkv.mkv_compress_params(self.B, wl.window, wl.sink, wl.keep_window, 1, 1, 1, 1e-6)
        self.dp = mkv.mkv_decode_params(1, 1, 1e-6)
        self.cache = mkv.alloc_cache(self.g, self.cap, dev)
        self.mom = mkv.alloc_moments(self.g, dev)
        self.ws_c = mkv.alloc_workspace(mkv.mkv_compress_workspace_size(self.g, self.T, self.p), dev)
        self.ws_d = mkv.alloc_workspace(mkv.mkv_decode_workspace_size(self.g, self.cap), dev)
        self.ws_e = mkv.alloc_workspace(mkv.mkv_evict_workspace_size(self.g, self.cap), dev)
        self.out = torch.empty(self.S, G.batch, G.n_q_heads, G.head_dim, device=dev)
        self.out_host = torch.empty(self.out.shape, dtype=torch.float32).pin_memory()
        self.stream = torch.cuda.Stream(dev)
        self.launches_per_step = 8 + self.S + self.S // EVICT_EVERY

    # the three parts as plain C-ABI calls on the current stream
    def compress(self):
        d = self.dev_in
        self.mkv.mkv_compress(self.g, self.T, d["K"], d["V"], d["Q"], self.p, self.cache, self.mom, self.ws_c)

    def decode(self, s):
        d = self.dev_in
        self.mkv.mkv_decode_step(self.g, d["q"][s], d["kn"][s], d["vn"][s], self.cache, self.mom, self.dp,
                                 self.out[s], None, self.ws_d)

    def evict(self, s):
        self.mkv.mkv_evict_append(self.g, self.dev_in["q"][s], None, None, self.B, self.cache, self.mom, 1e-6,
                                  self.ws_e)

    def eager_step(self):
        self.compress()
        for s in range(self.S):
            self.decode(s)
            if (s + 1) % EVICT_EVERY == 0:
                self.evict(s)

    def capture(self):
        torch = self.t
        with torch.cuda.stream(self.stream):
            self.eager_step()  # warm: function attributes, SM-count cache
        self.stream.synchronize()
        self.graphs = []
        def cap(fn):
            gr = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gr, stream=self.stream, capture_error_mode="relaxed"):
                fn()
            return gr
        self.g_compress = cap(self.compress)
        self.g_blocks = []
        for b0 in range(0, self.S, EVICT_EVERY):
            gd = cap(lambda b0=b0: [self.decode(s) for s in range(b0, min(self.S, b0 + EVICT_EVERY))])
            ge = cap(lambda b0=b0: self.evict(min(self.S, b0 + EVICT_EVERY) - 1))
            self.g_blocks.append((gd, ge))

    def replay(self, ev=None):
        """Replays one step on self.stream; ev: list of 2 + 2*blocks events to record between parts."""
        torch = self.t
        with torch.cuda.stream(self.stream):
            if ev:
                ev[0].record(self.stream)
            self.g_compress.replay()
            k = 1
            if ev:
                ev[k].record(self.stream)
            for gd, ge in self.g_blocks:
                gd.replay()
                k += 1
                if ev:
                    ev[k].record(self.stream)
                ge.replay()
                k += 1
                if ev:
                    ev[k].record(self.stream)

    def n_events(self):
        return 2 + 2 * len(self.g_blocks)

    def check_errors(self):
        for ws in (self.ws_c, self.ws_d, self.ws_e):
            code, info = self.mkv.mkv_get_device_error(ws, self.stream)
            if code != 0:
                raise RuntimeError(f"device error {code} (unit {info})")

    # algorithmic bytes: every input read once, every output written once
    def decode_bytes_total(self):
        G, d = self.G, self.G.head_dim
        units = G.batch * G.n_kv_heads
        tot = 0
        length = self.B
        for s in range(self.S):
            tot += units * (length * d * 2 * 2 + d * d * 4 + 2 * d * 4 + 4)   # retained K,V + moments
            tot += G.batch * G.n_q_heads * d * 2 + units * d * 2 * 2            # q, k_new/v_new
            tot += units * d * 2 * 2 + G.batch * G.n_q_heads * d * 4            # appended row, out
            length += 1
            if (s + 1) % EVICT_EVERY == 0:
                length = self.B
        return tot

    def compress_bytes(self):
        G, d = self.G, self.G.head_dim
        units = G.batch * G.n_kv_heads
        return units * (2 * self.T * d * 2 + G.group * self.wl.window * d * 2 + self.B * d * 2 * 2
                        + (d * d + 2 * d + 1) * 4)


def l2_flush(torch, buf):
    buf.zero_()


def run_gpu(args):
    import torch
    from paper_2606_01563_gb300 import inputs, mkv
    rank, world, local = dist_env()
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    mkv.lib()
    if args.only:
        hbm, _ = peaks()
        flush = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device=dev)
        legs = {"decode_sweep": lambda: decode_sweep(torch, mkv, dev, flush, hbm),
                "compress_long": lambda: compress_long(torch, mkv, inputs, dev, flush, hbm),
                "continuous_eviction": lambda: continuous_eviction(torch, mkv, dev),
                "layers_one_launch": lambda: layers_one_launch(torch, mkv, dev, flush, hbm)}
        print(json.dumps({"only": args.only, args.only: legs[args.only]()}), flush=True)
        return
    step = Step(torch, mkv, inputs, seed=1000 * rank, dev=dev)
    step.capture()
    flush = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device=dev)
    st = step.stream

    for _ in range(args.warmup):
        l2_flush(torch, flush)
        step.replay()
    st.synchronize()
    step.check_errors()

    # ---- device-timed steps
    nev = step.n_events()
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(nev)] for _ in range(args.steps)]
    clocks = Clocks(local)
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    clocks.start()
    for k in range(args.steps):
        with torch.cuda.stream(st):
            l2_flush(torch, flush)
        step.replay(evs[k])
    st.synchronize()
    torch.cuda.synchronize()
    clk = clocks.stop()
    if dist:
        dist.barrier()
    step.check_errors()
    seg = np.array([[evs[k][i].elapsed_time(evs[k][i + 1]) for i in range(nev - 1)] for k in range(args.steps)])
    step_ms = seg.sum(axis=1)
    compress_ms = seg[:, 0]
    decode_ms = seg[:, 1::2].sum(axis=1)
    evict_ms = seg[:, 2::2].sum(axis=1)
    ms_per_step, value = job_throughput(float(step_ms.sum()), args.steps, step.G.batch * step.S, dist, dev)

    # ---- end to end: host inputs in, decode outputs back, inside the timed region
    e2e_ms = []
    h2d = sum(v.numel() * v.element_size() for v in step.host_in.values())
    d2h = step.out.numel() * 4
    for k in range(max(3, min(args.steps, 10))):
        l2_flush(torch, flush)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(st):
            e0.record(st)
            for name, hv in step.host_in.items():
                step.dev_in[name].copy_(hv, non_blocking=True)
        step.replay()
        with torch.cuda.stream(st):
            step.out_host.copy_(step.out, non_blocking=True)
            e1.record(st)
        st.synchronize()
        e2e_ms.append(e0.elapsed_time(e1))
    e2e_step, e2e_value = job_throughput(float(np.sum(e2e_ms)), len(e2e_ms), step.G.batch * step.S, dist, dev)

    # ---- roofline of the dominant kernel
    hbm, peak_kind = peaks()
    dec_launch_ms = float(decode_ms.mean()) / step.S
    dec_bytes = step.decode_bytes_total() / step.S
    cmp_bytes = step.compress_bytes()
    shares = {"decode": float(decode_ms.mean() / step_ms.mean()), "compress": float(compress_ms.mean() / step_ms.mean()),
              "evict": float(evict_ms.mean() / step_ms.mean())}
    dominant = max(shares, key=shares.get)
    if dominant == "decode":
        achieved = dec_bytes / (dec_launch_ms / 1e3) / 1e9
        src = kernel_sources("decode.cu")
        kern = "decode_kernel"
    elif dominant == "compress":
        achieved = cmp_bytes / (float(compress_ms.mean()) / 1e3) / 1e9
        src = kernel_sources("compress.cu")
        kern = "compress (8 launches)"
    else:
        achieved = None
        src = kernel_sources("evict.cu")
        kern = "evict_kernel"
    tr = NCU_TRAFFIC.get(dominant)
    traffic = tr["bytes"] if tr and tr.get("code_sha") == code_sha(src) else None
    roof = {"kernel": kern, "bound": "hbm", "achieved": None if achieved is None else round(achieved, 1),
            "peak": hbm, "peak_kind": peak_kind, "unit": "GB/s",
            "frac": None if achieved is None else round(achieved / hbm, 4), "traffic": traffic,
            "algorithmic_bytes_per_launch": dec_bytes if dominant == "decode" else cmp_bytes,
            "shares": {k: round(v, 4) for k, v in shares.items()}}

    line = {"metric": METRIC, "value": round(value, 2), "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(ms_per_step, 4), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": f"{WORKLOAD}: Llama-3.1-8B attention geometry, 1 layer, batch 1, "
                                   f"32 q heads / 8 kv heads, d=128, T=8192, budget 512, window 32, sink 1, "
                                   f"mi on, 256 decode steps with append, evict every {EVICT_EVERY}",
                       "global_batch": step.G.batch * world, "seq_len": step.T, "decode_steps": step.S,
                       "parallelism": f"replicas x{world}", "accum": "f32", "l2": "flushed (256 MB write) "
                       "before every timed step", "graphs": "one CUDA graph per part, replayed"},
            "e2e": {"value": round(e2e_value, 2), "unit": "tokens/s", "h2d_bytes_per_step": int(h2d),
                    "d2h_bytes_per_step": int(d2h), "ms_per_step": round(e2e_step, 4)},
            "gpu_launches": step.launches_per_step * args.steps,
            "parts_ms": {"compress": round(float(compress_ms.mean()), 4), "decode_256": round(float(decode_ms.mean()), 4),
                         "evict_4": round(float(evict_ms.mean()), 4)},
            "decode": {"avg_launch_us": round(dec_launch_ms * 1e3, 3), "gbs": round(dec_bytes / dec_launch_ms / 1e6, 1),
                       "frac": round(dec_bytes / dec_launch_ms / 1e6 / hbm, 4)},
            "compress": {"gbs": round(cmp_bytes / float(compress_ms.mean()) / 1e6, 1)},
            "roofline": roof, "clocks": clk}
    if rank == 0 and not args.no_extras:
        line["decode_sweep"] = decode_sweep(torch, mkv, dev, flush, hbm)
        line["compress_long"] = compress_long(torch, mkv, inputs, dev, flush, hbm)
        line["continuous_eviction"] = continuous_eviction(torch, mkv, dev)
        line["layers_one_launch"] = layers_one_launch(torch, mkv, dev, flush, hbm)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline()
    if dist:
        dist.barrier()
        dist.destroy_process_group()
    if rank == 0:
        print(json.dumps(line), flush=True)


def decode_sweep(torch, mkv, dev, flush, hbm):
    """Decode throughput cells: batch x budget on the Llama geometry, dense fp32 C,
    correction on/off.  Each cell is timed two ways: one launch alone with L2
    flushed before it (graph launch included), and the steady state over many
    layers' caches (decode_layers)."""
    res = []
    H, G, D = 8, 4, 128
    gen = torch.Generator(device=dev)
    gen.manual_seed(5)
    st = torch.cuda.Stream(dev)
    for b in (1, 8, 32, 64):
        for B in (256, 1024, 4096):
            g = mkv.geom(b, H, G, D)
            cap = B
            cache = mkv.Cache(torch.randn(b, H, cap, D, device=dev, generator=gen).bfloat16(),
                              torch.randn(b, H, cap, D, device=dev, generator=gen).bfloat16(),
                              torch.zeros(b, H, cap, dtype=torch.int32, device=dev),
                              torch.full((b, H), B, dtype=torch.int32, device=dev),
                              torch.full((b, H), B, dtype=torch.int32, device=dev))
            mom = mkv.Moments(torch.full((b, H), 8192, dtype=torch.int32, device=dev),
                              0.05 * torch.randn(b, H, D, device=dev, generator=gen),
                              0.05 * torch.randn(b, H, D, device=dev, generator=gen),
                              0.05 * torch.randn(b, H, D, D, device=dev, generator=gen))
            q = torch.randn(b, H * G, D, device=dev, generator=gen).bfloat16()
            out = torch.empty(b, H * G, D, device=dev)
            ws = mkv.alloc_workspace(mkv.mkv_decode_workspace_size(g, cap), dev)
            cell = {"batch": b, "budget": B}
            for corr in (1, 0):
                p = mkv.mkv_decode_params(corr, 1, 1e-6)
                with torch.cuda.stream(st):
                    mkv.mkv_decode_step(g, q, None, None, cache, mom, p, out, None, ws, st)
                    gr = torch.cuda.CUDAGraph()
                with torch.cuda.graph(gr, stream=st, capture_error_mode="relaxed"):
                    mkv.mkv_decode_step(g, q, None, None, cache, mom, p, out, None, ws, st)
                times = []
                for it in range(12):
                    with torch.cuda.stream(st):
                        flush.zero_()
                        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                        e0.record(st)
                        gr.replay()
                        e1.record(st)
                    st.synchronize()
                    if it >= 2:
                        times.append(e0.elapsed_time(e1))
                t = float(np.median(times))
                units = b * H
                byt = units * (B * D * 4 + (D * D * 4 + 2 * D * 4 + 4 if corr else 0)) + b * H * G * D * (2 + 4)
                key = "corr" if corr else "plain"
                cell[key] = {"us": round(t * 1e3, 2), "gbs": round(byt / t / 1e6, 1),
                             "frac": round(byt / t / 1e6 / hbm, 4), "tokens_per_s": round(b / (t / 1e3), 1)}
            code, _ = mkv.mkv_get_device_error(ws, st)
            cell["ok"] = code == 0
            del cache, mom, ws
            cell.update(decode_layers(torch, mkv, dev, flush, hbm, b, B, gen, st))
            res.append(cell)
    return res


def decode_layers(torch, mkv, dev, flush, hbm, b, B, gen, st):
    """Steady-state decode as in a model: one launch per layer, each layer with
    its own cache and moments, the layers' bytes together at least twice the
    L2 (so every launch reads HBM), back to back in one CUDA graph; L2 flushed
    before every replay.  Per-launch time = replay time / layers."""
    H, G, D = 8, 4, 128
    g = mkv.geom(b, H, G, D)
    units = b * H
    per_layer = units * (B * D * 4 + D * D * 4 + 2 * D * 4 + 4) + b * H * G * D * (2 + 4)
    layers = int(min(256, max(4, -(-2 * 129 * 2 ** 20 // per_layer))))
    Kall = torch.randn(layers, b, H, B, D, device=dev, generator=gen).bfloat16()
    Vall = torch.randn(layers, b, H, B, D, device=dev, generator=gen).bfloat16()
    Call = 0.05 * torch.randn(layers, b, H, D, D, device=dev, generator=gen)
    mk = 0.05 * torch.randn(layers, b, H, D, device=dev, generator=gen)
    mv = 0.05 * torch.randn(layers, b, H, D, device=dev, generator=gen)
    n = torch.full((layers, b, H), 8192, dtype=torch.int32, device=dev)
    pos = torch.zeros(b, H, B, dtype=torch.int32, device=dev)
    lens = torch.full((b, H), B, dtype=torch.int32, device=dev)
    seen = torch.full((b, H), B, dtype=torch.int32, device=dev)
    q = torch.randn(b, H * G, D, device=dev, generator=gen).bfloat16()
    out = torch.empty(b, H * G, D, device=dev)
    ws = mkv.alloc_workspace(mkv.mkv_decode_workspace_size(g, B), dev)
    caches = [mkv.Cache(Kall[l], Vall[l], pos, lens, seen) for l in range(layers)]
    moms = [mkv.Moments(n[l], mk[l], mv[l], Call[l]) for l in range(layers)]
    # the 16-bit moment storage of Sec. C.2: a bf16 copy of every layer's C
    C16 = torch.empty(layers, b, H, D, D, dtype=torch.bfloat16, device=dev)
    for l in range(layers):
        mkv.mkv_moments_pack_bf16(g, moms[l], C16[l])
    res = {}
    for corr in (1, 0, 2):
        p = mkv.mkv_decode_params(min(corr, 1), 1, 1e-6)
        ps = [p] * layers
        if corr == 2:
            ps = [mkv.mkv_decode_params(1, 1, 1e-6, C16[l].data_ptr()) for l in range(layers)]
        with torch.cuda.stream(st):
            for l in range(layers):
                mkv.mkv_decode_step(g, q, None, None, caches[l], moms[l], ps[l], out, None, ws, st)
            gr = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gr, stream=st, capture_error_mode="relaxed"):
            for l in range(layers):
                mkv.mkv_decode_step(g, q, None, None, caches[l], moms[l], ps[l], out, None, ws, st)
        times = []
        for it in range(6):
            with torch.cuda.stream(st):
                flush.zero_()
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record(st)
                gr.replay()
                e1.record(st)
            st.synchronize()
            if it >= 2:
                times.append(e0.elapsed_time(e1) / layers)
        t = float(np.median(times))
        cbytes = {0: 0, 1: D * D * 4 + 2 * D * 4 + 4, 2: D * D * 2 + 2 * D * 4 + 4}[corr]
        byt = units * (B * D * 4 + cbytes) + b * H * G * D * (2 + 4)
        res[{0: "plain", 1: "corr", 2: "corr_c16"}[corr] + "_layers"] = {
            "us": round(t * 1e3, 2), "gbs": round(byt / t / 1e6, 1), "frac": round(byt / t / 1e6 / hbm, 4),
            "tokens_per_s": round(b / (t / 1e3), 1), "layers": layers}
        del gr
    code, _ = mkv.mkv_get_device_error(ws, st)
    res["ok_layers"] = code == 0
    del Kall, Vall, Call, C16, caches, moms
    return res


def layers_one_launch(torch, mkv, dev, flush, hbm, layers=32, B=512):
    """Decode for all 32 layers of the Llama-3.1-8B geometry at batch 1 (budget
    512, correction on), two ways: the layers' caches, moments and queries
    stacked on the batch dimension and decoded by one launch, and one launch
    per layer back to back in a graph.  The single launch applies where the
    layers' queries are available together (independent per-layer state, no
    cross-layer dependency inside the step)."""
    H, G, D = 8, 4, 128
    gen = torch.Generator(device=dev).manual_seed(9)
    rnd = lambda *shape: torch.randn(*shape, device=dev, generator=gen)
    K, V = rnd(layers, H, B, D).bfloat16(), rnd(layers, H, B, D).bfloat16()
    C, mk, mv = 0.05 * rnd(layers, H, D, D), 0.05 * rnd(layers, H, D), 0.05 * rnd(layers, H, D)
    n = torch.full((layers, H), 8192, dtype=torch.int32, device=dev)
    pos = torch.zeros(layers, H, B, dtype=torch.int32, device=dev)
    lens = torch.full((layers, H), B, dtype=torch.int32, device=dev)
    q = rnd(layers, H * G, D).bfloat16()
    out = torch.empty(layers, H * G, D, device=dev)
    p = mkv.mkv_decode_params(1, 1, 1e-6)
    st = torch.cuda.Stream(dev)
    gall, g1 = mkv.geom(layers, H, G, D), mkv.geom(1, H, G, D)
    ws_all = mkv.alloc_workspace(mkv.mkv_decode_workspace_size(gall, B), dev)
    ws_1 = mkv.alloc_workspace(mkv.mkv_decode_workspace_size(g1, B), dev)
    stacked = (mkv.Cache(K, V, pos, lens, lens.clone()), mkv.Moments(n, mk, mv, C))
    per = [(mkv.Cache(K[l:l + 1], V[l:l + 1], pos[l:l + 1], lens[l:l + 1], lens[l:l + 1].clone()),
            mkv.Moments(n[l:l + 1], mk[l:l + 1], mv[l:l + 1], C[l:l + 1])) for l in range(layers)]
    res = {"layers": layers, "batch": 1, "budget": B}
    for mode in ("one_launch", "per_layer"):
        def body():
            if mode == "one_launch":
                mkv.mkv_decode_step(gall, q, None, None, stacked[0], stacked[1], p, out, None, ws_all, st)
            else:
                for l in range(layers):
                    mkv.mkv_decode_step(g1, q[l:l + 1], None, None, per[l][0], per[l][1], p, out[l:l + 1], None,
                                        ws_1, st)
        with torch.cuda.stream(st):
            body()
            gr = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gr, stream=st, capture_error_mode="relaxed"):
            body()
        times = []
        for it in range(10):
            with torch.cuda.stream(st):
                flush.zero_()
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record(st)
                gr.replay()
                e1.record(st)
            st.synchronize()
            if it >= 2:
                times.append(e0.elapsed_time(e1))
        t = float(np.median(times))
        byt = layers * H * (B * D * 4 + D * D * 4 + 2 * D * 4 + 4) + layers * H * G * D * (2 + 4)
        res[mode] = {"us": round(t * 1e3, 2), "gbs": round(byt / t / 1e6, 1), "frac": round(byt / t / 1e6 / hbm, 4)}
        del gr
    res["ok"] = all(mkv.mkv_get_device_error(w, st)[0] == 0 for w in (ws_all, ws_1))
    return res


def continuous_eviction(torch, mkv, dev, steps=64):
    """Algorithm 1 once per generated token with the cache at its budget (one
    append and one eviction per step, Llama-3.1-8B geometry, budget 512):
    mkv_decode_evict_step, and the two calls it stands for (mkv_evict_append,
    then mkv_decode_step), each as a graph of `steps` steps."""
    res = []
    for b in (1, 8):
        H, G, D, B, cap = 8, 4, 128, 512, 576
        g = mkv.geom(b, H, G, D)
        gen = torch.Generator(device=dev).manual_seed(3)
        rnd = lambda *shape: torch.randn(*shape, device=dev, generator=gen)
        K0, V0 = rnd(b, H, cap, D).bfloat16(), rnd(b, H, cap, D).bfloat16()
        qs, kn, vn = rnd(steps, b, H * G, D).bfloat16(), rnd(steps, b, H, D).bfloat16(), rnd(steps, b, H, D).bfloat16()
        mom0 = (0.05 * rnd(b, H, D), 0.05 * rnd(b, H, D), 0.01 * rnd(b, H, D, D))
        out = torch.empty(b, H * G, D, device=dev)
        p = mkv.mkv_decode_params(1, 1, 1e-6)
        st = torch.cuda.Stream(dev)
        cell = {"batch": b, "budget": B}
        for mode in ("one_call", "two_calls"):
            cache = mkv.Cache(K0.clone(), V0.clone(),
                              torch.arange(cap, dtype=torch.int32, device=dev).expand(b, H, cap).contiguous(),
                              torch.full((b, H), B, dtype=torch.int32, device=dev),
                              torch.full((b, H), 10 ** 4, dtype=torch.int32, device=dev))
            mom = mkv.Moments(torch.full((b, H), 7000, dtype=torch.int32, device=dev), *(x.clone() for x in mom0))
            wsf = mkv.alloc_workspace(mkv.mkv_decode_evict_workspace_size(g, cap), dev)
            wse = mkv.alloc_workspace(mkv.mkv_evict_workspace_size(g, cap), dev)
            wsd = mkv.alloc_workspace(mkv.mkv_decode_workspace_size(g, cap), dev)

            def body():
                for i in range(steps):
                    if mode == "one_call":
                        mkv.mkv_decode_evict_step(g, qs[i], kn[i], vn[i], B, cache, mom, p, out, None, wsf, st)
                    else:
                        mkv.mkv_evict_append(g, qs[i], kn[i], vn[i], B, cache, mom, 1e-6, wse, st)
                        mkv.mkv_decode_step(g, qs[i], None, None, cache, mom, p, out, None, wsd, st)
            with torch.cuda.stream(st):
                body()
                st.synchronize()
                gr = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gr, stream=st, capture_error_mode="relaxed"):
                body()
            times = []
            for it in range(4):
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                with torch.cuda.stream(st):
                    e0.record(st)
                    gr.replay()
                    e1.record(st)
                st.synchronize()
                if it >= 1:
                    times.append(e0.elapsed_time(e1) * 1e3 / steps)
            ok = all(mkv.mkv_get_device_error(w, st)[0] == 0 for w in (wsf, wse, wsd))
            cell[mode] = {"us_per_step": round(float(np.median(times)), 2),
                          "tokens_per_s": round(b * 1e6 / float(np.median(times)), 1), "ok": ok}
            del gr, cache, mom, wsf, wse, wsd
        res.append(cell)
        torch.cuda.empty_cache()
    return res


def compress_long(torch, mkv, inputs, dev, flush, hbm):
    """Compress throughput at 32K (Qwen3-4B geometry, batch 4, budget 1024) and 128K
    (Llama-3.1-8B geometry, batch 1, budget 128, window 64) context, one layer;
    ms_adaptive is the same compression with the budget shared by the KV heads
    of each batch item."""
    res = {}
    st = torch.cuda.Stream(dev)
    for name in ("qwen4b_t32k", "llama8b_t128k"):
        wl = inputs.WORKLOADS[name]
        G = wl.geom
        g = mkv.geom(G.batch, G.n_kv_heads, G.group, G.head_dim)
        gen = inputs.Generator(wl, seed=11)
        K, V, Q = gen.prefill()
        tb = inputs.to_bf16_tensor
        K, V, Q = tb(K).to(dev), tb(V).to(dev), tb(Q).to(dev)
        prot = 1 + wl.window
        for adaptive in (0, 1):
            p = mkv.mkv_compress_params(wl.budget, wl.window, 1, 1, 1, 1, 1, 1e-6, adaptive)
            cap = min(wl.T, G.n_kv_heads * (wl.budget - prot) + prot) if adaptive else wl.budget + EVICT_EVERY
            cache, mom = mkv.alloc_cache(g, cap, dev), mkv.alloc_moments(g, dev)
            ws = mkv.alloc_workspace(mkv.mkv_compress_workspace_size(g, wl.T, p), dev)
            times = []
            for it in range(5):
                with torch.cuda.stream(st):
                    flush.zero_()
                    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                    e0.record(st)
                    mkv.mkv_compress(g, wl.T, K, V, Q, p, cache, mom, ws, stream=st)
                    e1.record(st)
                st.synchronize()
                if it >= 1:
                    times.append(e0.elapsed_time(e1))
            code, _ = mkv.mkv_get_device_error(ws, st)
            t = float(np.median(times))
            if adaptive:  # the budget shared by the KV heads of each batch item
                res[name]["ms_adaptive"] = round(t, 3)
                res[name]["ok"] = res[name]["ok"] and code == 0
            else:
                units = G.batch * G.n_kv_heads
                byt = units * 2 * wl.T * G.head_dim * 2
                flops = units * (2 * G.group * wl.window * wl.T * G.head_dim + 4 * wl.T * G.head_dim ** 2)
                res[name] = {"T": wl.T, "batch": G.batch, "budget": wl.budget, "ms": round(t, 3),
                             "gbs": round(byt / t / 1e6, 1), "frac_hbm": round(byt / t / 1e6 / hbm, 4),
                             "tflops": round(flops / t / 1e9, 2), "ok": code == 0}
            del cache, mom, ws
        del K, V, Q
        torch.cuda.empty_cache()
    return res


# --------------------------------------------------------------------------
# the oracle on the host cores
# --------------------------------------------------------------------------
def oracle_sample(inputs, O, seed, unit):
    """One KV-head unit of the bench step through the fp64 oracle; returns seconds (wall, cpu)."""
    wl = inputs.WORKLOADS[WORKLOAD]
    G = wl.geom
    gen = inputs.Generator(wl, seed=seed)
    K, V, Q = gen.prefill()
    q, kn, vn = gen.decode(wl.decode_steps)
    bi, h = divmod(unit, G.n_kv_heads)
    t0, c0 = time.perf_counter(), resource.getrusage(resource.RUSAGE_SELF)
    ref = O.compress(K[bi, h], V[bi, h], Q[bi, h], wl.budget, wl.window, wl.sink, True, 1, True, 1e-6)
    Kr, Vr, m, pos = K[bi, h][ref.idx], V[bi, h][ref.idx], ref.moments, np.array(ref.idx)
    for s in range(wl.decode_steps):
        qh = q[s, bi, h * G.group:(h + 1) * G.group]
        _, _, Kr, Vr = O.decode_step(qh, Kr, Vr, m, kn[s, bi, h], vn[s, bi, h], tau=1e-6)
        pos = np.append(pos, wl.T + s)
        if (s + 1) % EVICT_EVERY == 0:
            ev = O.evict_append(qh, Kr, Vr, pos, m, wl.budget, 1e-6)
            Kr, Vr, m, pos = ev.K, ev.V, ev.moments, ev.pos
    t1, c1 = time.perf_counter(), resource.getrusage(resource.RUSAGE_SELF)
    cpu = (c1.ru_utime - c0.ru_utime) + (c1.ru_stime - c0.ru_stime)
    return t1 - t0, cpu


def cpu_baseline():
    import oracle as O
    from paper_2606_01563_gb300 import inputs
    wl = inputs.WORKLOADS[WORKLOAD]
    units = wl.geom.batch * wl.geom.n_kv_heads
    wall, cpu = 0.0, 0.0
    n = 0
    t_start = time.perf_counter()
    while n < units and (n < 2 or time.perf_counter() - t_start < 20.0):
        w, c = oracle_sample(inputs, O, 0, n)
        wall += w
        cpu += c
        n += 1
    est = wall / n * units
    tokens = wl.geom.batch * wl.decode_steps
    return {"value": round(tokens / est, 3), "unit": "tokens/s", "cores": max(1, round(cpu / wall)),
            "kind": "oracle", "sample": f"{n} of {units} KV-head units of the full step (compress T=8192, "
            f"256 decode steps, 4 evictions), fp64 numpy, scaled by {units}/{n}; "
            f"{wall:.1f} s wall, host nproc={os.cpu_count()}; cores = CPU time / wall time (numpy's BLAS threads)"}


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    import oracle as O
    from paper_2606_01563_gb300 import inputs
    wl = inputs.WORKLOADS[WORKLOAD]
    units = wl.geom.batch * wl.geom.n_kv_heads
    for k in range(args.warmup):
        oracle_sample(inputs, O, 0, k % units)
    wall, cpu = 0.0, 0.0
    for k in range(args.steps):
        w, c = oracle_sample(inputs, O, 0, k % units)
        wall += w
        cpu += c
    est_ms = wall / args.steps * units * 1e3
    tokens = wl.geom.batch * wl.decode_steps
    value = tokens / (est_ms / 1e3)
    cores = max(1, round(cpu / wall))
    sample = (f"each step: one of {units} KV-head units of the full step (compress T=8192, 256 decode steps, "
              f"4 evictions) through the fp64 oracle, scaled by {units}; cores = CPU time / wall time")
    print(json.dumps({"impl": "reference", "metric": METRIC, "value": round(value, 3), "unit": "tokens/s",
                      "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(est_ms, 2),
                      "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
                      "data": "synthetic", "config": {"workload": WORKLOAD, "seq_len": wl.T,
                                                      "decode_steps": wl.decode_steps},
                      "cpu_baseline": {"value": round(value, 3), "unit": "tokens/s", "cores": cores,
                                       "kind": "oracle", "sample": sample},
                      "e2e": {"value": round(value, 3), "unit": "tokens/s", "h2d_bytes_per_step": 0,
                              "d2h_bytes_per_step": 0}}), flush=True)


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
