"""mkv_decode_step_noalloc: the decode entry point for callers that cannot
allocate device memory (an engine plugin handed only its input and output
buffers, a server whose memory is reserved up front, a path that cannot take
cudaMalloc's device synchronisation).  Its scratch is the library's fixed
device array.  Two calls in a row must match the workspace entry point,
mkv_decode_step, on identical inputs within the decode tolerance, and
oversized geometries must be rejected.  This file is collected last so that
a stop-at-first-failure run has already run every other test."""
import numpy as np
import pytest
import torch

from paper_2606_01563_gb300 import mkv
from paper_2606_01563_gb300.inputs import bf16_round
from gpu_util import assert_output_close, bf16, f32, host, i32

pytestmark = pytest.mark.gpu


def make(rng, b, H, D, cap, lens):
    K = bf16(bf16_round(rng.standard_normal((b, H, cap, D))))
    V = bf16(bf16_round(rng.standard_normal((b, H, cap, D))))
    return lambda: mkv.Cache(K.clone(), V.clone(), i32(np.zeros((b, H, cap))), i32(lens), i32(lens))


def test_noalloc_matches_workspace_entry_point():
    rng = np.random.default_rng(77)
    b, H, G, D, cap = 2, 8, 4, 128, 600
    g = mkv.geom(b, H, G, D)
    lens = rng.integers(100, cap - 4, (b, H)).astype(np.int32)
    fresh = make(rng, b, H, D, cap, lens)
    cache_ws, cache_na = fresh(), fresh()
    mom = mkv.Moments(i32(rng.integers(1, 9000, (b, H))), f32(0.3 * rng.standard_normal((b, H, D))),
                      f32(0.3 * rng.standard_normal((b, H, D))), f32(0.05 * rng.standard_normal((b, H, D, D))))
    p = mkv.mkv_decode_params(1, 1, 1e-6)
    ws = mkv.alloc_workspace(mkv.mkv_decode_workspace_size(g, cap))
    for call in range(2):
        q = bf16(bf16_round(2.0 * rng.standard_normal((b, H * G, D))))
        kn = bf16(bf16_round(rng.standard_normal((b, H, D))))
        vn = bf16(bf16_round(rng.standard_normal((b, H, D))))
        out_ws = torch.empty(b, H * G, D, device="cuda")
        out_na = torch.full((b, H * G, D), float("nan"), device="cuda")
        lse_ws = torch.empty(b, H * G, device="cuda")
        lse_na = torch.empty(b, H * G, device="cuda")
        mkv.mkv_decode_step(g, q, kn, vn, cache_ws, mom, p, out_ws, lse_ws, ws)
        mkv.mkv_decode_step_noalloc(g, q, kn, vn, cache_na, mom, p, out_na, lse_na)
        torch.cuda.synchronize()
        assert_output_close(host(out_na), host(out_ws), f"call {call}")
        np.testing.assert_allclose(host(lse_na), host(lse_ws), rtol=0, atol=1e-4)
        np.testing.assert_array_equal(host(cache_na.len), host(cache_ws.len))
        np.testing.assert_array_equal(host(cache_na.K), host(cache_ws.K))
    assert mkv.mkv_get_device_error(ws)[0] == 0


def test_noalloc_rejects_oversized_geometry():
    g = mkv.geom(1024, 8, 8, 128)  # one partial per query head alone exceeds the 4 MiB scratch
    cache = mkv.alloc_cache(mkv.geom(1, 1, 1, 128), 4)
    p = mkv.mkv_decode_params(0, 1, 0.0)
    out = torch.empty(1, device="cuda")
    with pytest.raises(mkv.MKVError) as e:
        mkv.mkv_decode_step_noalloc(g, out, None, None, cache, None, p, out, None)
    assert e.value.code == 7


def _oracle_decode(q, K, V, lens, n, mu_k, mu_v, C, kn, vn, G, tau=1e-6):
    import oracle as O
    b, H = lens.shape
    D = K.shape[-1]
    out = np.zeros((b, H * G, D))
    lse = np.zeros((b, H * G))
    for bi in range(b):
        for h in range(H):
            L = lens[bi, h]
            m = O.Moments(int(n[bi, h]), mu_k[bi, h], mu_v[bi, h], C[bi, h])
            o, l, _, _ = O.decode_step(q[bi, h * G:(h + 1) * G], K[bi, h, :L], V[bi, h, :L], m, kn[bi, h], vn[bi, h],
                                       True, 1, tau)
            out[bi, h * G:(h + 1) * G] = o
            lse[bi, h * G:(h + 1) * G] = l
    return out, lse


def _case(rng, b, H, G, D, cap):
    """Host arrays of one decode call (cache, moments, query, new token)."""
    K = bf16_round(rng.standard_normal((b, H, cap, D)))
    V = bf16_round(rng.standard_normal((b, H, cap, D)))
    lens = rng.integers(1, cap - 1, (b, H)).astype(np.int32)
    n = rng.integers(0, 5000, (b, H)).astype(np.int32)
    mu_k = (0.3 * rng.standard_normal((b, H, D))).astype(np.float32)
    mu_v = (0.3 * rng.standard_normal((b, H, D))).astype(np.float32)
    C = (0.05 * rng.standard_normal((b, H, D, D))).astype(np.float32)
    q = bf16_round(2.0 * rng.standard_normal((b, H * G, D)))
    kn = bf16_round(rng.standard_normal((b, H, D)))
    vn = bf16_round(rng.standard_normal((b, H, D)))
    return dict(K=K, V=V, lens=lens, n=n, mu_k=mu_k, mu_v=mu_v, C=C, q=q, kn=kn, vn=vn, cap=cap)


def _noalloc_vs_oracle(c, b, H, G, D, what):
    g = mkv.geom(b, H, G, D)
    cache = mkv.Cache(bf16(c["K"]), bf16(c["V"]), i32(np.zeros((b, H, c["cap"]))), i32(c["lens"]), i32(c["lens"]))
    mom = mkv.Moments(i32(c["n"]), f32(c["mu_k"]), f32(c["mu_v"]), f32(c["C"]))
    out = torch.full((b, H * G, D), float("nan"), device="cuda")
    lse = torch.full((b, H * G), float("nan"), device="cuda")
    mkv.mkv_decode_step_noalloc(g, bf16(c["q"]), bf16(c["kn"]), bf16(c["vn"]), cache, mom,
                                mkv.mkv_decode_params(1, 1, 1e-6), out, lse)
    torch.cuda.synchronize()
    want, want_lse = _oracle_decode(c["q"], c["K"], c["V"], c["lens"], c["n"], c["mu_k"], c["mu_v"], c["C"], c["kn"],
                                    c["vn"], G)
    assert_output_close(host(out), want, what)
    np.testing.assert_allclose(host(lse), want_lse, rtol=1e-4, atol=1e-4)
    np.testing.assert_array_equal(host(cache.len), c["lens"] + 1)


def test_noalloc_against_oracle_alternating_geometries():
    """A geometry with few units and one with many, alternating, each call
    against the fp64 oracle: one call's partial records must not disturb the
    next call's ticket counters or results (the counters sit in a region of
    their own in the shared array)."""
    rng = np.random.default_rng(78)
    small = (1, 2, 2, 64, 200)
    large = (8, 8, 4, 128, 700)   # 64 units, two splits each
    for k, geom in enumerate([small, large, small, large]):
        b, H, G, D, cap = geom
        _noalloc_vs_oracle(_case(rng, b, H, G, D, cap), b, H, G, D, f"call {k} geometry {geom}")


def test_noalloc_near_largest_accepted_geometry():
    """1024 units (one split each: more units than SMs), about half of the
    fixed scratch.  With at most two CTAs per SM per launch the split count
    times the units never exceeds twice the SM count, so the partial records
    stay far below the array's size (at most 304 x 8 x 132 floats) and every
    accepted geometry runs with its full split count; the size check rejects
    by units (the f_hat rows)."""
    rng = np.random.default_rng(79)
    b, H, G, D, cap = 16, 64, 4, 64, 40
    _noalloc_vs_oracle(_case(rng, b, H, G, D, cap), b, H, G, D, "1024 units")


def test_noalloc_ticket_merge_alternating_geometries():
    """The merge through the array's partial records and ticket counters (the
    variant for clusters that cannot be co-scheduled, forced by a test hook),
    alternating a geometry with few units and one with many: the counters a
    call leaves at zero must still be zero for the next call, whatever the
    previous call's partial records overwrote."""
    rng = np.random.default_rng(80)
    small = (1, 2, 2, 64, 200)
    large = (8, 8, 4, 128, 700)
    prev = mkv.mkv_debug_force_ticket_merge(1)
    try:
        for k, geom in enumerate([large, small, large, small, large]):
            b, H, G, D, cap = geom
            _noalloc_vs_oracle(_case(rng, b, H, G, D, cap), b, H, G, D, f"ticket call {k} geometry {geom}")
    finally:
        mkv.mkv_debug_force_ticket_merge(prev)
