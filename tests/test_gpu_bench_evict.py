"""The benchmark's own periodic eviction, checked against the fp64 oracle on
every unit: the one-layer Llama-3.1-8B workload of the bench (T = 8192,
budget 512, window 32, the bench's device-drawn inputs), compressed, 64
decode steps that each append a token (576 rows), then one mkv_evict_append
back to the budget: 64 evictions in one call, 8 units.  The calls are the
bench's own (bench.Stack and bench.Run, run eagerly instead of from graphs),
so the decode steps read C' in the operand form the run packs.

The oracle starts from the state the compress left (checked first against the
oracle's compress, near ties continued from the kernel's choice), checks
every decode step's output, and follows the kernel's 64 evictions (each the
argmin of Algorithm 1's scores under the state reached, or at a near tie one
of the near-minimal rows), then compares the surviving rows and moments."""
import os
import sys

import numpy as np
import pytest
import torch

import oracle as O
from paper_2606_01563_gb300 import inputs, mkv
from gpu_util import assert_output_close, host
from parity import check_compress_unit, check_evicted_unit, evicted_moments

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402

TAU = 1e-6


def test_bench_periodic_eviction_all_units():
    dev = torch.device("cuda", 0)
    wl = inputs.WORKLOADS["llama8b_layer_t8k"]
    every = 64
    stack = bench.Stack(torch, inputs, wl, seed=7, dev=dev, layers=1, steps=every)
    run = bench.Run(torch, mkv, stack, wl.budget, every, dev)
    G_, T, B = wl.geom, wl.T, wl.budget
    H, G = G_.n_kv_heads, G_.group
    # the compress the bench times, with its diagnostics
    s = torch.zeros(1, H, T, device=dev)
    s2 = torch.zeros_like(s)
    i1 = torch.zeros(1, H, B, dtype=torch.int32, device=dev)
    mkv.mkv_compress(run.g, T, stack.K[0], stack.V[0], stack.Q[0], run.p, run.caches[0], run.moms[0], run.ws_c,
                     diag=(s, s2, i1))
    # the run's decode steps read C' in its operand form: packed after every
    # compress and eviction, as the run's own compress does
    mkv.mkv_moments_pack_split(run.g, run.moms[0], TAU, run.csplit[0])
    c, m = run.caches[0], run.moms[0]
    comp = dict(K=host(c.K), V=host(c.V), pos=host(c.pos), len=host(c.len), seen=host(c.seen), n=host(m.n),
                mu_k=host(m.mu_k), mu_v=host(m.mu_v), C=host(m.C), s=host(s), s2=host(s2), i1=host(i1))
    K, V, Q = (host(x)[0] for x in (stack.K[0], stack.V[0], stack.Q[0]))
    q, kn, vn = (host(x)[:, 0, 0] for x in (stack.q, stack.kn, stack.vn))   # [steps, heads, d]
    state = {}
    for h in range(H):
        check_compress_unit(comp, 0, h, K[h], V[h], Q[h], T, B, wl.window, wl.sink, bool(wl.keep_window), 1, 1, TAU)
        R = comp["pos"][0, h, :B]
        state[h] = dict(K=K[h][R], V=V[h][R], pos=R.astype(np.int64), m=evicted_moments(K[h], V[h], R))
    # 64 decode steps with append, then the eviction, as the bench runs them
    for i in range(every):
        run.decode(stack, i)
    run.evict(stack, every - 1)
    code, info = mkv.mkv_get_device_error(run.ws_d)
    assert code == 0, (code, info)
    code, info = mkv.mkv_get_device_error(run.ws_e)
    assert code == 0, (code, info)
    outs = host(run.final)[:, 0]   # [steps, q heads, d]
    c, m = run.caches[0], run.moms[0]
    got = dict(K=host(c.K), V=host(c.V), pos=host(c.pos), len=host(c.len), seen=host(c.seen), n=host(m.n),
               mu_k=host(m.mu_k), mu_v=host(m.mu_v), C=host(m.C))
    ties = 0
    for h in range(H):
        st = state[h]
        Kr, Vr, pos = st["K"], st["V"], st["pos"]
        for i in range(every):
            qh = q[i, h * G:(h + 1) * G]
            o, _, Kr, Vr = O.decode_step(qh, Kr, Vr, st["m"], kn[i, h], vn[i, h], True, 1, TAU)
            pos = np.append(pos, T + i)
            assert_output_close(outs[i, h * G:(h + 1) * G], o, f"decode step {i} unit {h}")
        assert got["seen"][0, h] == T + every
        f = check_evicted_unit(got, 0, h, q[every - 1, h * G:(h + 1) * G], Kr, Vr, pos, st["m"], B, TAU)
        assert len(f.pos) == B
        ties += f.ties
    print(f"near ties met over the 8 units' 64 evictions: {ties}")
