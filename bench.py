"""Benchmark of the MomentKV hot path on GB300.

Workload (the headline line): the Qwen3-4B attention geometry, all 36 layers
(32 query heads, 8 KV heads, d=128, bf16), batch 4 at context 32768, window
32, one sink, moment filter on, at each of the budgets 128, 256 and 1024.
A step runs, for each budget in turn, one compress of every layer's prompt,
then 512 decode steps; a decode step is one corrected decode launch per
layer, layer after layer, each appending that step's token.  So a step is
3 x (36 compressions + 18432 decode launches) and generates 3 x 4 x 512
tokens.  Prompts (19.3 GB over the 36 layers) and per-step queries and new
tokens are synthetic, drawn on the device (inputs.TorchGenerator), resident
in HBM before the timed region.  Each part is captured once in a CUDA graph
and replayed; CUDA events on the launching stream time the parts.  L2 is
flushed (a 256 MB write) before every timed step, outside the timed region.

value      generated decode tokens per second of whole-step time (device-timed).
e2e        the same with every input of the step (the 36 prompts, queries and
           new tokens) copied from pinned host memory, and the last layer's
           output of every decode step copied back, inside the timed region;
           steps are pipelined over two device input sets, so one step's
           copies run while the step before it computes.
roofline   the dominant kernel against the measured HBM copy bandwidth.
extra keys the Llama-3.1-8B 32-layer 128K workload (budget 128, window 64,
           1024 decode steps, an evict-append on every layer every 64
           tokens), the one-layer Llama-3.1-8B 8K workload, the decode sweep
           cells (batch x budget, correction on/off), compress with the
           budget shared across heads, the continuous eviction mode, and 32
           layers' decode in one launch against one launch per layer.

--impl reference times the fp64 oracle on the host cores instead: each step
is a bounded sample of the same workload (16 (layer, unit, budget) jobs run
by a process pool), reported as the throughput that sample implies.
--only LEG runs one of the extra legs alone and prints its result, so that a
profiler can capture that leg without the headline's launches.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import multiprocessing as mp
import os
import resource
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "decode-step attn+correction tokens/s and HBM GB/s frac; compress GB/s at 1 GB300"
HEADLINE = "qwen4b_t32k"
BUDGETS = (128, 256, 1024)
TAU = 1e-6
ORACLE_JOBS = 16  # (layer, unit, budget) jobs in one oracle sample

# dram__bytes_read.sum + dram__bytes_write.sum per launch of a kernel on the
# headline workload from one ncu capture, valid while the code the kernel
# compiles from (its .cu file and the library headers, comments aside) is
# what was captured: code_sha of those sources at capture time.
NCU_TRAFFIC = {"decode_cl_kernel": {"bytes": 15292836,
                                     "code_sha": "9d69462747c1f8bffb7c37fcf5df73f0f2a83953d0808a02ddcb68ad837127a8"}}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--no-extras", action="store_true", help="skip the extra legs")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true", help="skip the end-to-end measurement")
    ap.add_argument("--layers", type=int, default=None, help="layers of the headline workload (default: all 36)")
    ap.add_argument("--only", choices=["t128k", "t8k", "decode_sweep", "compress_adaptive", "continuous_eviction",
                                       "layers_one_launch"],
                    help="run one extra leg alone and print its result (for profiling that leg)")
    return ap.parse_args()


def config_dict(layers=None):
    """The workload description both arms print."""
    from paper_2606_01563_gb300 import inputs
    wl = inputs.WORKLOADS[HEADLINE]
    L = wl.n_layers if layers is None else layers
    return {"workload": f"{HEADLINE}: Qwen3-4B attention geometry, {L} layers, batch 4, 32 q heads / 8 kv heads, "
                        f"d=128, T=32768, budgets 128/256/1024 in turn, window 32, sink 1, mi on; per budget: "
                        f"compress every layer, then 512 decode steps (one launch per layer, append)",
            "layers": L, "global_batch": wl.geom.batch, "seq_len": wl.T, "budgets": list(BUDGETS),
            "decode_steps": wl.decode_steps, "parallelism": "replicas", "accum": "f32",
            "l2": "flushed (256 MB write) before every timed step; a step reads >19 GB"}


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
    return [os.path.join(c, cu), os.path.join(c, "common.cuh"), os.path.join(c, "warp_mma.cuh"),
            os.path.join(c, "kernels.h"), os.path.join(ROOT, "include", "mkv.h")]


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
# a multi-layer workload on the device
# --------------------------------------------------------------------------
class Stack:
    """Device inputs of a multi-layer workload: each layer's prompt K, V,
    Q_obs, and each (decode step, layer)'s query and new token, drawn on the
    device by inputs.TorchGenerator (one generator per layer)."""

    def __init__(self, torch, inputs, wl, seed, dev, layers=None, steps=None):
        G = wl.geom
        self.wl, self.G = wl, G
        self.L = wl.n_layers if layers is None else layers
        self.S = wl.decode_steps if steps is None else steps
        d = G.head_dim
        bf = torch.bfloat16
        self.K, self.V, self.Q = [], [], []
        self.q = torch.empty(self.S, self.L, G.batch, G.n_q_heads, d, dtype=bf, device=dev)
        self.kn = torch.empty(self.S, self.L, G.batch, G.n_kv_heads, d, dtype=bf, device=dev)
        self.vn = torch.empty_like(self.kn)
        for l in range(self.L):
            gen = inputs.TorchGenerator(wl, seed=seed, layer=l, device=dev)
            K, V, Q = gen.prefill()
            self.K.append(K)
            self.V.append(V)
            self.Q.append(Q)
            q, kn, vn = gen.decode(self.S)
            self.q[:, l] = q
            self.kn[:, l] = kn
            self.vn[:, l] = vn
            del gen
        torch.cuda.synchronize(dev)

    def tensors(self):
        return self.K + self.V + self.Q + [self.q, self.kn, self.vn]

    def twin(self):
        """A second set of device input buffers of the same shapes (contents
        copied from this one), for double-buffered end-to-end steps."""
        t = object.__new__(Stack)
        t.wl, t.G, t.L, t.S = self.wl, self.G, self.L, self.S
        t.K = [x.clone() for x in self.K]
        t.V = [x.clone() for x in self.V]
        t.Q = [x.clone() for x in self.Q]
        t.q, t.kn, t.vn = self.q.clone(), self.kn.clone(), self.vn.clone()
        return t

    def nbytes(self):
        return sum(t.numel() * t.element_size() for t in self.tensors())


class Run:
    """One budget of a multi-layer workload on a Stack: compress every layer,
    then `steps` decode steps, each one mkv_decode_step per layer (layer
    after layer, appending the step's token), and an mkv_evict_append on
    every layer back to the budget every `evict_every` steps (0: never)."""

    def __init__(self, torch, mkv, stack, budget, evict_every, dev):
        self.t, self.mkv, self.st = torch, mkv, stack
        wl, G = stack.wl, stack.G
        self.G, self.B, self.ev_every = G, budget, evict_every
        self.g = mkv.geom(G.batch, G.n_kv_heads, G.group, G.head_dim)
        self.cap = budget + (evict_every if evict_every else stack.S)
        self.p = mkv.mkv_compress_params(budget, wl.window, wl.sink, wl.keep_window, wl.pool, 1, 1, TAU)
        # with periodic eviction the caches keep y_j = S_tilde k_j across calls
        self.caches = [mkv.alloc_cache(self.g, self.cap, dev, evict_state=bool(evict_every)) for _ in range(stack.L)]
        self.moms = [mkv.alloc_moments(self.g, dev) for _ in range(stack.L)]
        # each layer's C' in the decode's operand form (bf16 hi, lo words),
        # packed whenever the layer's moments change (compress, eviction)
        d = G.head_dim
        self.csplit = [torch.empty(G.batch, G.n_kv_heads, d, d, dtype=torch.int32, device=dev) for _ in range(stack.L)]
        # a layer chain: the kernel before each decode launch belongs to another
        # layer (or is a compress, pack or eviction of another layer), so the
        # launch may read its cache and moments before its dependency wait
        early = 1 if stack.L > 1 else 0
        self.dps = [mkv.mkv_decode_params(1, 1, TAU, None, early, c.data_ptr()) for c in self.csplit]
        # one workspace per kind, shared by the layers (the calls run one after another on one stream)
        self.ws_c = mkv.alloc_workspace(mkv.mkv_compress_workspace_size(self.g, wl.T, self.p), dev)
        self.ws_d = mkv.alloc_workspace(mkv.mkv_decode_workspace_size(self.g, self.cap), dev)
        self.ws_e = mkv.alloc_workspace(mkv.mkv_evict_workspace_size(self.g, self.cap), dev) if evict_every else None
        self.out = torch.empty(G.batch, G.n_q_heads, G.head_dim, device=dev)        # a layer's output
        self.final = torch.empty(stack.S, G.batch, G.n_q_heads, G.head_dim, device=dev)  # last layer's, per step
        self.block = evict_every if evict_every else 64

    def compress(self, s):
        for l in range(s.L):
            self.mkv.mkv_compress(self.g, s.wl.T, s.K[l], s.V[l], s.Q[l], self.p, self.caches[l], self.moms[l],
                                  self.ws_c)
            self.mkv.mkv_moments_pack_split(self.g, self.moms[l], TAU, self.csplit[l])

    def decode(self, s, i):
        for l in range(s.L):
            out = self.final[i] if l == s.L - 1 else self.out
            self.mkv.mkv_decode_step(self.g, s.q[i, l], s.kn[i, l], s.vn[i, l], self.caches[l], self.moms[l],
                                     self.dps[l], out, None, self.ws_d)

    def evict(self, s, i):
        for l in range(s.L):
            self.mkv.mkv_evict_append(self.g, s.q[i, l], None, None, self.B, self.caches[l], self.moms[l], TAU,
                                      self.ws_e)
            self.mkv.mkv_moments_pack_split(self.g, self.moms[l], TAU, self.csplit[l])

    def parts(self, s):
        """(kind, callable) in step order, reading the inputs of stack `s`."""
        out = [("compress", lambda: self.compress(s))]
        for b0 in range(0, s.S, self.block):
            b1 = min(s.S, b0 + self.block)
            out.append(("decode", lambda b0=b0, b1=b1: [self.decode(s, i) for i in range(b0, b1)]))
            if self.ev_every and b1 % self.ev_every == 0:
                out.append(("evict", lambda i=b1 - 1: self.evict(s, i)))
        return out

    def capture(self, stream, stack=None):
        """Capture the parts over `stack`'s inputs (default: the run's own
        stack) as one more graph set; the first set is self.graphs."""
        torch = self.t
        s = self.st if stack is None else stack
        with torch.cuda.stream(stream):
            for _, fn in self.parts(s):  # warm: function attributes, SM-count cache
                fn()
        stream.synchronize()
        graphs = []
        for kind, fn in self.parts(s):
            gr = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gr, stream=stream, capture_error_mode="relaxed"):
                fn()
            graphs.append((kind, gr))
        if not hasattr(self, "graph_sets"):
            self.graph_sets = []
        self.graph_sets.append(graphs)
        self.graphs = self.graph_sets[0]

    def launches(self):
        """Kernels of ours one pass launches (9 per per-unit compress, one
        pack of C' after each compress and eviction)."""
        s = self.st
        n_ev = (s.S // self.ev_every) if self.ev_every else 0
        return s.L * (9 + 1 + s.S + 2 * n_ev)

    def check_errors(self, stream):
        for ws in (self.ws_c, self.ws_d, self.ws_e):
            if ws is None:
                continue
            code, info = self.mkv.mkv_get_device_error(ws, stream)
            if code != 0:
                raise RuntimeError(f"device error {code} (unit {info}) at budget {self.B}")

    # algorithmic bytes: every input read once, every output written once
    def decode_bytes(self):
        """Total over the pass's decode launches."""
        G, d, s = self.G, self.G.head_dim, self.st
        units = G.batch * G.n_kv_heads
        tot, length = 0, self.B
        for i in range(s.S):
            per = units * (length * d * 2 * 2 + d * d * 4 + 2 * d * 4 + 4)    # retained K,V + moments
            per += G.batch * G.n_q_heads * d * 2 + units * d * 2 * 2          # q, k_new/v_new
            per += units * d * 2 * 2 + G.batch * G.n_q_heads * d * 4          # appended row, out
            tot += per * s.L
            length += 1
            if self.ev_every and (i + 1) % self.ev_every == 0:
                length = self.B
        return tot

    def compress_bytes(self):
        """Algorithmic bytes of one layer's compress: K and V read once, window queries, outputs written once."""
        G, d, wl = self.G, self.G.head_dim, self.st.wl
        units = G.batch * G.n_kv_heads
        return units * (2 * wl.T * d * 2 + G.group * wl.window * d * 2 + self.B * (d * 2 * 2 + 4)
                        + (d * d + 2 * d + 1) * 4)

    def compress_flops(self):
        G, d, wl = self.G, self.G.head_dim, self.st.wl
        units = G.batch * G.n_kv_heads
        return units * (2 * G.group * wl.window * wl.T * d + 4 * wl.T * d * d)


def replay(runs, stream, ev=None):
    """One step: every run's parts in order on `stream`; ev[k] recorded before
    part k and after the last one."""
    torch = runs[0].t
    k = 0
    with torch.cuda.stream(stream):
        for r in runs:
            for _, gr in r.graphs:
                if ev is not None:
                    ev[k].record(stream)
                gr.replay()
                k += 1
        if ev is not None:
            ev[k].record(stream)


def part_kinds(runs):
    return [(r.B, kind) for r in runs for kind, _ in r.graphs]


def time_steps(torch, runs, stream, flush, steps):
    """Device time of `steps` steps, L2 flushed before each: per-part times [steps, parts] (ms)."""
    nparts = sum(len(r.graphs) for r in runs)
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(nparts + 1)] for _ in range(steps)]
    for k in range(steps):
        with torch.cuda.stream(stream):
            flush.zero_()
        replay(runs, stream, evs[k])
    stream.synchronize()
    return np.array([[evs[k][i].elapsed_time(evs[k][i + 1]) for i in range(nparts)] for k in range(steps)])


def summarise(runs, seg, hbm):
    """Per budget and kind: ms per step, and the decode / compress roofline figures."""
    kinds = part_kinds(runs)
    res = {}
    for r in runs:
        cols = {kind: [i for i, (B, k) in enumerate(kinds) if B == r.B and k == kind] for kind in
                ("compress", "decode", "evict")}
        ms = {k: float(seg[:, c].sum(axis=1).mean()) if c else 0.0 for k, c in cols.items()}
        n_dec = r.st.S * r.st.L
        dec_b = r.decode_bytes()
        L = r.st.L
        res[r.B] = {"ms": {k: round(v, 4) for k, v in ms.items()},
                    "decode": {"launches": n_dec, "avg_launch_us": round(ms["decode"] * 1e3 / n_dec, 3),
                               "bytes_per_launch": round(dec_b / n_dec), "gbs": round(dec_b / ms["decode"] / 1e6, 1),
                               "frac": round(dec_b / ms["decode"] / 1e6 / hbm, 4)},
                    "compress": {"ms_per_layer": round(ms["compress"] / L, 4),
                                 "gbs": round(r.compress_bytes() * L / ms["compress"] / 1e6, 1),
                                 "frac": round(r.compress_bytes() * L / ms["compress"] / 1e6 / hbm, 4),
                                 "tflops": round(r.compress_flops() * L / ms["compress"] / 1e9, 2)},
                    "decode_bytes": dec_b}
        if r.ev_every:
            n_ev = (r.st.S // r.ev_every) * L
            res[r.B]["evict"] = {"launches": n_ev, "avg_launch_us": round(ms["evict"] * 1e3 / max(1, n_ev), 2)}
    return res


def l2_flush_buffer(torch, dev):
    return torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device=dev)


def e2e_measure(torch, stacks, runs, stream, steps):
    """End to end through the C ABI, steps pipelined over two input sets.
    Every input of a step (the prompts, queries and new tokens) is copied
    from pinned host memory on a copy stream, into the set the step reads,
    while the previous step computes; each budget's last-layer outputs are
    copied back on a third stream after that budget's decode (the budget's
    next decode waits for that read).  The timed region runs from the first
    input copy to the last output read.  Each run holds one graph set per
    input set.  Returns (total ms, h2d bytes per step, d2h bytes per step,
    per-step copy ms)."""
    dev = stream.device
    sets = [s.tensors() for s in stacks]
    host_in = []
    for t in sets[0]:
        h = torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
        h.copy_(t)
        host_in.append(h)
    host_out = [torch.empty(r.final.shape, dtype=r.final.dtype, pin_memory=True) for r in runs]
    up, down = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    Ev = torch.cuda.Event
    ready = [Ev(), Ev()]
    free, read = [None, None], [None] * len(runs)
    copies = []

    def load(k):  # one step's inputs into set k, once the step before that used set k is done
        if free[k] is not None:
            up.wait_event(free[k])
        c0, c1 = Ev(enable_timing=True), Ev(enable_timing=True)
        with torch.cuda.stream(up):
            c0.record(up)
            for d, h in zip(sets[k], host_in):
                d.copy_(h, non_blocking=True)
            c1.record(up)
            ready[k].record(up)
        copies.append((c0, c1))

    torch.cuda.synchronize(dev)
    e0, e1 = Ev(enable_timing=True), Ev(enable_timing=True)
    e0.record(up)
    load(0)
    for i in range(steps):
        k = i % 2
        if i + 1 < steps:
            load(1 - k)
        stream.wait_event(ready[k])
        for j, r in enumerate(runs):
            if read[j] is not None:
                stream.wait_event(read[j])
            with torch.cuda.stream(stream):
                for _, gr in r.graph_sets[k]:
                    gr.replay()
                done = Ev()
                done.record(stream)
            down.wait_event(done)
            with torch.cuda.stream(down):
                host_out[j].copy_(r.final, non_blocking=True)
                read[j] = Ev()
                read[j].record(down)
        free[k] = Ev()
        free[k].record(stream)
    with torch.cuda.stream(down):
        down.wait_event(free[(steps - 1) % 2])
        e1.record(down)
    torch.cuda.synchronize(dev)
    h2d = sum(t.numel() * t.element_size() for t in host_in)
    d2h = sum(t.numel() * t.element_size() for t in host_out)
    copy_ms = [c0.elapsed_time(c1) for c0, c1 in copies]
    del host_in, host_out
    return e0.elapsed_time(e1), h2d, d2h, copy_ms


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
    hbm, peak_kind = peaks()
    flush = l2_flush_buffer(torch, dev)
    if args.only:
        legs = {"t128k": lambda: leg_t128k(torch, mkv, inputs, dev, flush, hbm),
                "t8k": lambda: leg_t8k(torch, mkv, inputs, dev, flush, hbm),
                "decode_sweep": lambda: decode_sweep(torch, mkv, dev, flush, hbm),
                "compress_adaptive": lambda: compress_adaptive(torch, mkv, inputs, dev, flush, hbm),
                "continuous_eviction": lambda: continuous_eviction(torch, mkv, dev),
                "layers_one_launch": lambda: layers_one_launch(torch, mkv, dev, flush, hbm)}
        print(json.dumps({"only": args.only, args.only: legs[args.only]()}), flush=True)
        return

    wl = inputs.WORKLOADS[HEADLINE]
    t_setup = time.perf_counter()
    stack = Stack(torch, inputs, wl, seed=1000 * rank, dev=dev, layers=args.layers)
    runs = [Run(torch, mkv, stack, B, 0, dev) for B in BUDGETS]
    stream = torch.cuda.Stream(dev)
    for r in runs:
        r.capture(stream)
    setup_s = time.perf_counter() - t_setup

    for _ in range(args.warmup):
        with torch.cuda.stream(stream):
            flush.zero_()
        replay(runs, stream)
    stream.synchronize()
    for r in runs:
        r.check_errors(stream)

    # ---- device-timed steps
    clocks = Clocks(local)
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    clocks.start()
    seg = time_steps(torch, runs, stream, flush, args.steps)
    torch.cuda.synchronize()
    clk = clocks.stop()
    if dist:
        dist.barrier()
    for r in runs:
        r.check_errors(stream)
    step_ms = seg.sum(axis=1)
    tokens = sum(stack.G.batch * stack.S for _ in runs)
    ms_per_step, value = job_throughput(float(step_ms.sum()), args.steps, tokens, dist, dev)
    per_budget = summarise(runs, seg, hbm)

    # ---- end to end through the C ABI
    e2e = None
    if not args.no_e2e:
        try:
            twin = stack.twin()
            for r in runs:
                r.capture(stream, twin)
            with torch.cuda.stream(stream):  # the second set's graphs once, untimed
                for r in runs:
                    for _, gr in r.graph_sets[1]:
                        gr.replay()
            stream.synchronize()
            for r in runs:
                r.check_errors(stream)
            e2e_steps = max(3, args.steps)
            total, h2d, d2h, copy_ms = e2e_measure(torch, [stack, twin], runs, stream, e2e_steps)
            for r in runs:
                r.check_errors(stream)
            e2e_step, e2e_value = job_throughput(total, e2e_steps, tokens, dist, dev)
            e2e = {"value": round(e2e_value, 2), "unit": "tokens/s", "h2d_bytes_per_step": int(h2d),
                   "d2h_bytes_per_step": int(d2h), "ms_per_step": round(e2e_step, 4), "steps": e2e_steps,
                   "h2d_ms_per_step": round(float(np.mean(copy_ms)), 3),
                   "pipelining": "two input sets: step i+1's inputs are copied while step i computes; "
                                 "the timed region runs from step 0's first input copy to the last output read",
                   "l2": "not flushed between pipelined steps; a step reads >19 GB"}
            del twin
        except RuntimeError as exc:  # pinned host memory for every input could not be had
            e2e = {"value": None, "unit": "tokens/s", "error": str(exc)[:200]}

    # ---- roofline of the dominant kernel
    kinds = part_kinds(runs)
    tot = {k: float(seg[:, [i for i, (_, kk) in enumerate(kinds) if kk == k]].sum(axis=1).mean())
           for k in ("compress", "decode")}
    shares = {k: round(v / float(step_ms.mean()), 4) for k, v in tot.items()}
    dec_bytes = sum(per_budget[r.B]["decode_bytes"] for r in runs)
    dec_launches = sum(r.st.S * r.st.L for r in runs)
    cmp_bytes = sum(r.compress_bytes() * r.st.L for r in runs)
    if shares["decode"] >= shares["compress"]:
        kern, achieved = "decode_cl_kernel", dec_bytes / (tot["decode"] / 1e3) / 1e9
        per_launch, src = dec_bytes / dec_launches, kernel_sources("decode_cl.cu")
        avg_us = tot["decode"] * 1e3 / dec_launches
    else:
        kern, achieved = "compress (9 launches per layer)", cmp_bytes / (tot["compress"] / 1e3) / 1e9
        per_launch, src = cmp_bytes / (stack.L * len(runs)), kernel_sources("compress.cu")
        avg_us = tot["compress"] * 1e3 / (stack.L * len(runs))
    tr = NCU_TRAFFIC.get(kern)
    traffic = tr["bytes"] if tr and tr.get("code_sha") == code_sha(src) else None
    roof = {"kernel": kern, "bound": "hbm", "achieved": round(achieved, 1), "peak": hbm, "peak_kind": peak_kind,
            "unit": "GB/s", "frac": round(achieved / hbm, 4), "traffic": traffic,
            "algorithmic_bytes_per_launch": round(per_launch), "avg_launch_us": round(avg_us, 3),
            "shares": shares}
    for r in runs:
        per_budget[r.B].pop("decode_bytes")

    line = {"metric": METRIC, "value": round(value, 2), "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(ms_per_step, 4), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": dict(config_dict(stack.L), parallelism=f"replicas x{world}"),
            "graphs": "one CUDA graph per part (compress of all layers; 64 decode steps x all layers)",
            "moment_c": "fp32 C; after each compress a pack writes C' (clamped) as the decode's bf16 hi + lo operand "
                        "words, the same bytes and products as reading C",
            "e2e": e2e, "gpu_launches": sum(r.launches() for r in runs) * args.steps,
            "per_budget": {str(k): v for k, v in per_budget.items()},
            "roofline": roof, "clocks": clk, "setup_s": round(setup_s, 1),
            "input_bytes": stack.nbytes()}
    oracle_in = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        oracle_in = oracle_jobs_from_stack(stack, ORACLE_JOBS)
    del runs, stack
    torch.cuda.empty_cache()
    if rank == 0 and not args.no_extras:
        line["t128k"] = leg_t128k(torch, mkv, inputs, dev, flush, hbm)
        line["t8k"] = leg_t8k(torch, mkv, inputs, dev, flush, hbm)
        line["decode_sweep"] = decode_sweep(torch, mkv, dev, flush, hbm)
        line["compress_adaptive"] = compress_adaptive(torch, mkv, inputs, dev, flush, hbm)
        line["continuous_eviction"] = continuous_eviction(torch, mkv, dev)
        line["layers_one_launch"] = layers_one_launch(torch, mkv, dev, flush, hbm)
    if oracle_in is not None:
        line["cpu_baseline"] = cpu_baseline(oracle_in, wl, stack_layers=line["config"]["layers"])
    if dist:
        dist.barrier()
        dist.destroy_process_group()
    if rank == 0:
        print(json.dumps(line), flush=True)


def run_leg(torch, mkv, inputs, dev, flush, hbm, wl, budget, evict_every, layers=None, steps=None, timed=3):
    """One multi-layer workload at one budget, timed as the headline is."""
    stack = Stack(torch, inputs, wl, seed=7, dev=dev, layers=layers, steps=steps)
    run = Run(torch, mkv, stack, budget, evict_every, dev)
    stream = torch.cuda.Stream(dev)
    run.capture(stream)
    for _ in range(1):
        replay([run], stream)
    stream.synchronize()
    run.check_errors(stream)
    seg = time_steps(torch, [run], stream, flush, timed)
    run.check_errors(stream)
    res = summarise([run], seg, hbm)[budget]
    step = float(seg.sum(axis=1).mean())
    res.pop("decode_bytes")
    out = {"layers": stack.L, "batch": stack.G.batch, "T": wl.T, "budget": budget, "window": wl.window,
           "decode_steps": stack.S, "evict_every": evict_every, "ms_per_step": round(step, 3),
           "tokens_per_s": round(stack.G.batch * stack.S / (step / 1e3), 1), "steps_timed": timed, **res,
           "launches_per_step": run.launches()}
    del run, stack
    torch.cuda.empty_cache()
    return out


def leg_t128k(torch, mkv, inputs, dev, flush, hbm):
    """Llama-3.1-8B geometry, 32 layers, batch 1, T=131072, budget 128,
    window 64, mixture keys; 1024 decode steps with an evict-append on every
    layer every 64 tokens (the cache grows from 128 to 192 rows and back)."""
    wl = inputs.WORKLOADS["llama8b_t128k"]
    return run_leg(torch, mkv, inputs, dev, flush, hbm, wl, wl.budget, wl.evict_every)


def leg_t8k(torch, mkv, inputs, dev, flush, hbm):
    """Llama-3.1-8B geometry, one layer, batch 1, T=8192, budget 512, window
    32; 256 decode steps with an evict-append every 64 tokens."""
    wl = inputs.WORKLOADS["llama8b_layer_t8k"]
    return run_leg(torch, mkv, inputs, dev, flush, hbm, wl, wl.budget, 64, timed=10)


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
                p = mkv.mkv_decode_params(corr, 1, TAU)
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
        p = mkv.mkv_decode_params(min(corr, 1), 1, TAU)
        ps = [p] * layers
        if corr == 2:
            ps = [mkv.mkv_decode_params(1, 1, TAU, C16[l].data_ptr()) for l in range(layers)]
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
    p = mkv.mkv_decode_params(1, 1, TAU)
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
    mkv_decode_evict_step with the cache keeping y_j = S_tilde k_j across
    calls, the same without that state, and the two calls it stands for
    (mkv_evict_append, then mkv_decode_step), each as a graph of `steps`
    steps."""
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
        p = mkv.mkv_decode_params(1, 1, TAU)
        st = torch.cuda.Stream(dev)
        cell = {"batch": b, "budget": B}
        for mode in ("one_call_state", "one_call", "two_calls"):
            cache = mkv.Cache(K0.clone(), V0.clone(),
                              torch.arange(cap, dtype=torch.int32, device=dev).expand(b, H, cap).contiguous(),
                              torch.full((b, H), B, dtype=torch.int32, device=dev),
                              torch.full((b, H), 10 ** 4, dtype=torch.int32, device=dev))
            if mode == "one_call_state":
                cache.y = torch.zeros(b, H, cap, D, device=dev)
                cache.y_len = torch.zeros(b, H, dtype=torch.int32, device=dev)
            mom = mkv.Moments(torch.full((b, H), 7000, dtype=torch.int32, device=dev), *(x.clone() for x in mom0))
            wsf = mkv.alloc_workspace(mkv.mkv_decode_evict_workspace_size(g, cap), dev)
            wse = mkv.alloc_workspace(mkv.mkv_evict_workspace_size(g, cap), dev)
            wsd = mkv.alloc_workspace(mkv.mkv_decode_workspace_size(g, cap), dev)

            def body():
                for i in range(steps):
                    if mode in ("one_call", "one_call_state"):
                        mkv.mkv_decode_evict_step(g, qs[i], kn[i], vn[i], B, cache, mom, p, out, None, wsf, st)
                    else:
                        mkv.mkv_evict_append(g, qs[i], kn[i], vn[i], B, cache, mom, TAU, wse, st)
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


def compress_adaptive(torch, mkv, inputs, dev, flush, hbm):
    """One layer's compress at 32K (Qwen3-4B geometry, batch 4, budget 1024) and
    128K (Llama-3.1-8B geometry, batch 1, budget 128, window 64) context, with
    the budget per unit and (ms_adaptive) shared by the KV heads of each batch
    item (Ada-KV allocation)."""
    res = {}
    st = torch.cuda.Stream(dev)
    for name in ("qwen4b_t32k", "llama8b_t128k"):
        wl = inputs.WORKLOADS[name]
        G = wl.geom
        g = mkv.geom(G.batch, G.n_kv_heads, G.group, G.head_dim)
        K, V, Q = inputs.TorchGenerator(wl, seed=11, device=dev).prefill()
        prot = 1 + wl.window
        for adaptive in (0, 1):
            p = mkv.mkv_compress_params(wl.budget, wl.window, 1, 1, 1, 1, 1, TAU, adaptive)
            cap = min(wl.T, G.n_kv_heads * (wl.budget - prot) + prot) if adaptive else wl.budget + 64
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
def oracle_job(job):
    """One (layer, unit) of the headline workload at one budget through the
    fp64 oracle: compress the prompt, then the decode steps with append.
    Returns (wall s, CPU s) of this process."""
    import oracle as O
    K, V, Q, q, kn, vn, budget, window, sink, T = job
    w0, c0 = time.perf_counter(), time.process_time()
    ref = O.compress(K, V, Q, budget, window, sink, True, 1, True, TAU)
    Kr, Vr, m = K[ref.idx], V[ref.idx], ref.moments
    for s in range(q.shape[0]):
        _, _, Kr, Vr = O.decode_step(q[s], Kr, Vr, m, kn[s], vn[s], tau=TAU)
    return time.perf_counter() - w0, time.process_time() - c0


def _to_np(t):
    return t.float().cpu().numpy()


def oracle_jobs_from_stack(stack, n, step=0):
    """n oracle jobs on the bytes the GPU consumed: units and budgets rotate
    with `step`; layers run from 0."""
    G, wl = stack.G, stack.wl
    units = G.batch * G.n_kv_heads
    jobs = []
    for j in range(n):
        k = step * n + j
        u = k % units
        layer = (k // units) % stack.L
        B = BUDGETS[k % len(BUDGETS)]
        bi, h = divmod(u, G.n_kv_heads)
        g = G.group
        jobs.append((_to_np(stack.K[layer][bi, h]), _to_np(stack.V[layer][bi, h]), _to_np(stack.Q[layer][bi, h]),
                     _to_np(stack.q[:, layer, bi, h * g:(h + 1) * g]), _to_np(stack.kn[:, layer, bi, h]),
                     _to_np(stack.vn[:, layer, bi, h]), B, wl.window, wl.sink, wl.T))
    return jobs


def oracle_pool(n):
    """A spawn process pool of n single-threaded workers (numpy's BLAS held to
    one thread each, so that n jobs use n cores)."""
    keys = ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")
    old = {k: os.environ.get(k) for k in keys}
    for k in keys:
        os.environ[k] = "1"
    try:
        pool = mp.get_context("spawn").Pool(processes=n)
        pool.map(_noop, range(n))  # workers started and importing done before any timing
    finally:
        for k, v in old.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v
    return pool


def _noop(x):
    import oracle  # noqa: F401
    return x


def oracle_step(pool, jobs):
    """Runs the jobs on the pool; (wall s, CPU s summed over the workers)."""
    t0 = time.perf_counter()
    res = pool.map(oracle_job, jobs, chunksize=1)
    return time.perf_counter() - t0, sum(c for _, c in res)


def step_tokens_equiv(wl, layers, n_jobs):
    """Tokens a sample of n_jobs (layer, unit, budget) jobs stands for: the
    full step has layers x units jobs per budget, each budget producing
    batch x decode_steps tokens."""
    units = wl.geom.batch * wl.geom.n_kv_heads
    return n_jobs * wl.geom.batch * wl.decode_steps / (layers * units)


def cpu_baseline(jobs, wl, stack_layers):
    n = min(len(jobs), os.cpu_count() or 1)
    pool = oracle_pool(n)
    try:
        wall, cpu = oracle_step(pool, jobs)
    finally:
        pool.close()
        pool.join()
    tok = step_tokens_equiv(wl, stack_layers, len(jobs))
    return {"value": round(tok / wall, 3), "unit": "tokens/s", "cores": n, "kind": "oracle",
            "sample": f"{len(jobs)} (layer, unit, budget) jobs of the headline step on the bytes the GPU consumed "
                      f"(each: compress T={wl.T}, then {wl.decode_steps} decode steps), fp64 numpy, one job per "
                      f"worker process, {n} workers; stands for {tok:.1f} of the step's "
                      f"{len(BUDGETS) * wl.geom.batch * wl.decode_steps} tokens; {wall:.1f} s wall, "
                      f"{cpu:.1f} s CPU, host nproc={os.cpu_count()}"}


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    import torch
    from paper_2606_01563_gb300 import inputs
    wl = inputs.WORKLOADS[HEADLINE]
    layers = wl.n_layers if args.layers is None else args.layers
    n = min(ORACLE_JOBS, os.cpu_count() or 1)
    pool = oracle_pool(n)
    # one layer's inputs drawn on the host with the headline's recipe (the
    # values differ from the GPU arm's device draw, the distribution does not);
    # the sample's units and budgets rotate from step to step
    gen = inputs.TorchGenerator(wl, seed=0, layer=0, device="cpu")
    K, V, Q = gen.prefill()
    q, kn, vn = gen.decode(wl.decode_steps)

    class One:  # a one-layer stack view for oracle_jobs_from_stack
        pass
    st = One()
    st.G, st.wl, st.L = wl.geom, wl, 1
    st.K, st.V, st.Q = [K], [V], [Q]
    st.q, st.kn, st.vn = q[:, None], kn[:, None], vn[:, None]
    try:
        for k in range(args.warmup):
            oracle_step(pool, oracle_jobs_from_stack(st, n, step=k))
        walls, cpus = [], []
        for k in range(args.steps):
            jobs = oracle_jobs_from_stack(st, n, step=args.warmup + k)
            w, c = oracle_step(pool, jobs)
            walls.append(w)
            cpus.append(c)
    finally:
        pool.close()
        pool.join()
    ms_per_step = float(np.mean(walls)) * 1e3
    tok = step_tokens_equiv(wl, layers, n)
    value = tok / (ms_per_step / 1e3)
    sample = (f"each step: {n} (layer, unit, budget) jobs of the headline step (each: compress T={wl.T}, then "
              f"{wl.decode_steps} decode steps) through the fp64 oracle, one job per worker process, {n} workers, "
              f"standing for {tok:.2f} of the step's {len(BUDGETS) * wl.geom.batch * wl.decode_steps} tokens; "
              f"inputs drawn on the host with the same recipe; {float(np.sum(cpus)) / float(np.sum(walls)):.1f} "
              f"cores busy on average; host nproc={os.cpu_count()}")
    print(json.dumps({"impl": "reference", "metric": METRIC, "value": round(value, 3), "unit": "tokens/s",
                      "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_per_step, 2),
                      "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
                      "data": "synthetic", "config": dict(config_dict(layers), parallelism=f"replicas x{world}"),
                      "cpu_baseline": {"value": round(value, 3), "unit": "tokens/s", "cores": n,
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
