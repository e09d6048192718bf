"""Decode in a model's layer chain with early loads (mkv_decode_params.early_load
= 1): several layers' caches, each decode step one launch per layer, layer
after layer, each appending its token, back to back on one stream, so that
every launch starts while the previous layer's is still running and reads its
own cache and moments before its dependency wait.  Every output of every
launch against the fp64 oracle; also with the bf16 copy of C, batch 1 (many
splits) and the large-batch one-split case."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2606_01563_gb300 import mkv
from paper_2606_01563_gb300.inputs import bf16_round
from gpu_util import assert_output_close, bf16, f32, host, i32

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("b,H,G,D,L,lens,cap,c16,steps,graph", [
    (2, 8, 4, 128, 3, (300, 420), 440, False, 3, False),
    (1, 8, 4, 128, 4, (130, 510), 520, False, 3, False),
    (1, 8, 4, 128, 3, (200, 260), 270, True, 3, False),
    (24, 8, 2, 64, 2, (60, 90), 100, False, 3, False),
    # two layers, few units, back to back from a graph: the launch two back
    # in the stream is the same layer, so a launch must not start (and read
    # its cache early) before its predecessor's own predecessor has finished
    (4, 8, 4, 128, 2, (100, 300), 340, False, 24, True),
    (1, 8, 4, 128, 2, (500, 600), 640, False, 24, True),
    (1, 2, 4, 64, 2, (40, 90), 120, False, 24, True),
    # the headline geometry (32 units) at budget-1024 lengths: five or six
    # tiles per CTA, so stages are refilled while the chain runs
    (4, 8, 4, 128, 3, (1024, 1300), 1340, False, 6, True),
])
def test_layer_chain_early_load(b, H, G, D, L, lens, cap, c16, steps, graph):
    rng = np.random.default_rng(b * 1000 + L * 10 + D)
    layers = []
    for l in range(L):
        K = bf16_round(rng.standard_normal((b, H, cap, D)))
        V = bf16_round(rng.standard_normal((b, H, cap, D)))
        ln = rng.integers(lens[0], lens[1], (b, H)).astype(np.int32)
        n = rng.integers(0, 6000, (b, H)).astype(np.int32)
        mk = (0.3 * rng.standard_normal((b, H, D))).astype(np.float32)
        mv = (0.3 * rng.standard_normal((b, H, D))).astype(np.float32)
        C = (0.05 * rng.standard_normal((b, H, D, D))).astype(np.float32)
        if c16:
            C = bf16_round(C)  # the oracle sees what the bf16 copy holds
        layers.append(dict(K=K, V=V, len=ln, n=n, mu_k=mk, mu_v=mv, C=C))
    q = bf16_round(2.0 * rng.standard_normal((steps, L, b, H * G, D)))
    kn = bf16_round(rng.standard_normal((steps, L, b, H, D)))
    vn = bf16_round(rng.standard_normal((steps, L, b, H, D)))
    g = mkv.geom(b, H, G, D)
    dev = []
    for st in layers:
        cache = mkv.Cache(bf16(st["K"]), bf16(st["V"]), i32(np.zeros((b, H, cap))), i32(st["len"]),
                          i32(st["len"]))
        mom = mkv.Moments(i32(st["n"]), f32(st["mu_k"]), f32(st["mu_v"]), f32(st["C"]))
        C16 = None
        if c16:
            C16 = torch.empty(b, H, D, D, dtype=torch.bfloat16, device="cuda")
            mkv.mkv_moments_pack_bf16(g, mom, C16)
        dev.append((cache, mom, C16))
    qd, knd, vnd = bf16(q), bf16(kn), bf16(vn)
    outs = torch.full((steps, L, b, H * G, D), float("nan"), device="cuda")
    ws = mkv.alloc_workspace(mkv.mkv_decode_workspace_size(g, cap))
    torch.cuda.synchronize()
    stream = torch.cuda.Stream()

    def chain():
        for i in range(steps):
            for l in range(L):
                cache, mom, C16 = dev[l]
                p = mkv.mkv_decode_params(1, 1, 1e-6, None if C16 is None else C16.data_ptr(), 1)
                mkv.mkv_decode_step(g, qd[i, l], knd[i, l], vnd[i, l], cache, mom, p, outs[i, l], None, ws, stream)

    if graph:
        # launched back to back from a CUDA graph, as a serving loop would,
        # so that consecutive launches really overlap (host launches from
        # Python leave gaps between them); the graph is captured from a copy
        # of the initial cache lengths and replayed once
        lens0 = [d[0].len.clone() for d in dev]
        seen0 = [d[0].seen.clone() for d in dev]
        with torch.cuda.stream(stream):
            chain()  # warm-up: function attributes and split counts
        stream.synchronize()
        gr = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gr, stream=stream, capture_error_mode="relaxed"):
            chain()
        for d, l0, s0 in zip(dev, lens0, seen0):
            d[0].len.copy_(l0)
            d[0].seen.copy_(s0)
        torch.cuda.synchronize()
        with torch.cuda.stream(stream):
            gr.replay()
    else:
        with torch.cuda.stream(stream):
            chain()
    stream.synchronize()
    code, info = mkv.mkv_get_device_error(ws)
    assert code == 0, (code, info)
    got = host(outs)
    for l, st in enumerate(layers):
        for bi in range(b):
            for h in range(H):
                n0 = st["len"][bi, h]
                Kr, Vr = st["K"][bi, h, :n0], st["V"][bi, h, :n0]
                m = O.Moments(int(st["n"][bi, h]), st["mu_k"][bi, h], st["mu_v"][bi, h], st["C"][bi, h])
                for i in range(steps):
                    o, _, Kr, Vr = O.decode_step(q[i, l, bi, h * G:(h + 1) * G], Kr, Vr, m, kn[i, l, bi, h],
                                                 vn[i, l, bi, h], True, 1, 1e-6)
                    assert_output_close(got[i, l, bi, h * G:(h + 1) * G], o, f"step {i} layer {l} unit {(bi, h)}")
        np.testing.assert_array_equal(host(dev[l][0].len), st["len"] + steps)
