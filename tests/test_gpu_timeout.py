"""The bounded-wait failure path on the GPU, without a fault or a hang: with
the pipeline waits' poll limit set to zero (include/mkv_debug.h), the first
wait of every CTA gives up at once, so each call that has such waits records
MKV_ERR_TIMEOUT in its workspace's error word, drains the copies and
tensor-core operations it had in flight (with the full limit), frees its
tensor memory and returns.  The eviction kernels have no such waits and
complete normally.  After the limit is restored, the same calls on the same
device and context match the oracle again.  Also: the decode's merge through
global partial records (the variant for clusters that cannot be
co-scheduled), forced by the other test hook, against the oracle."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2606_01563_gb300 import mkv
from paper_2606_01563_gb300.inputs import WORKLOADS, Generator
from gpu_util import assert_output_close, bf16, host
from parity import check_compress_unit, evicted_moments

pytestmark = pytest.mark.gpu

TIMEOUT = 5


def _tiny_state():
    """A valid compressed tiny workload (cache at B + 1 rows of capacity B + 8)
    and one decode step's query and token."""
    wl = WORKLOADS["tiny_d64_t1k"]
    gen = Generator(wl, seed=3)
    K, V, Q = gen.prefill()
    q, kn, vn = gen.decode(1)
    G_ = wl.geom
    g = mkv.geom(G_.batch, G_.n_kv_heads, G_.group, G_.head_dim)
    T, B, cap = wl.T, wl.budget, wl.budget + 8
    p = mkv.mkv_compress_params(B, wl.window, wl.sink, wl.keep_window, 1, 1, 1, 1e-6)
    cache, mom = mkv.alloc_cache(g, cap), mkv.alloc_moments(g)
    ws = mkv.alloc_workspace(mkv.mkv_compress_workspace_size(g, T, p))
    mkv.mkv_compress(g, T, bf16(K), bf16(V), bf16(Q), p, cache, mom, ws)
    assert mkv.mkv_get_device_error(ws)[0] == 0
    return dict(wl=wl, g=g, p=p, K=K, V=V, Q=Q, q=q, kn=kn, vn=vn, cache=cache, mom=mom, cap=cap)


def _clone(st):
    c, m = st["cache"], st["mom"]
    return (mkv.Cache(c.K.clone(), c.V.clone(), c.pos.clone(), c.len.clone(), c.seen.clone()),
            mkv.Moments(m.n.clone(), m.mu_k.clone(), m.mu_v.clone(), m.C.clone()))


def _each_entry_point(st):
    """Each entry point once on valid inputs (a fresh copy of the compressed
    state, never the output of another call); status word of each."""
    wl, g, cap = st["wl"], st["g"], st["cap"]
    G_ = wl.geom
    codes = {}
    cache, mom = mkv.alloc_cache(g, cap), mkv.alloc_moments(g)
    ws = mkv.alloc_workspace(mkv.mkv_compress_workspace_size(g, wl.T, st["p"]))
    mkv.mkv_compress(g, wl.T, bf16(st["K"]), bf16(st["V"]), bf16(st["Q"]), st["p"], cache, mom, ws)
    codes["compress"] = mkv.mkv_get_device_error(ws)[0]
    out = torch.empty(G_.batch, G_.n_q_heads, G_.head_dim, device="cuda")
    dp = mkv.mkv_decode_params(1, 1, 1e-6)
    q, kn, vn = bf16(st["q"][0]), bf16(st["kn"][0]), bf16(st["vn"][0])
    cache, mom = _clone(st)
    ws = mkv.alloc_workspace(mkv.mkv_decode_workspace_size(g, cap))
    mkv.mkv_decode_step(g, q, kn, vn, cache, mom, dp, out, None, ws)
    codes["decode"] = mkv.mkv_get_device_error(ws)[0]
    cache, mom = _clone(st)
    ws = mkv.alloc_workspace(mkv.mkv_decode_evict_workspace_size(g, cap))
    mkv.mkv_decode_evict_step(g, q, kn, vn, wl.budget, cache, mom, dp, out, None, ws)
    codes["decode_evict"] = mkv.mkv_get_device_error(ws)[0]
    cache, mom = _clone(st)
    ws = mkv.alloc_workspace(mkv.mkv_evict_workspace_size(g, cap))
    mkv.mkv_evict_append(g, q, kn, vn, wl.budget - 2, cache, mom, 1e-6, ws)
    codes["evict"] = mkv.mkv_get_device_error(ws)[0]
    return codes


def test_timeouts_are_reported_then_calls_recover():
    st = _tiny_state()
    prev = mkv.mkv_debug_set_poll_limit(0)
    try:
        codes = _each_entry_point(st)
    finally:
        mkv.mkv_debug_set_poll_limit(-1)
    assert prev > 0
    assert codes == {"compress": TIMEOUT, "decode": TIMEOUT, "decode_evict": TIMEOUT, "evict": 0}, codes
    assert _each_entry_point(st) == {"compress": 0, "decode": 0, "decode_evict": 0, "evict": 0}
    # the context is still usable: a compress and a decode match the oracle
    # again (near ties continued from the kernel's choice)
    wl = WORKLOADS["tiny_d64_t1k"]
    gen = Generator(wl, seed=5)
    K, V, Q = gen.prefill()
    q, kn, vn = gen.decode(1)
    G_ = wl.geom
    H, G, T, B = G_.n_kv_heads, G_.group, wl.T, wl.budget
    g = mkv.geom(1, H, G, G_.head_dim)
    p = mkv.mkv_compress_params(B, wl.window, wl.sink, wl.keep_window, 1, 1, 1, 1e-6)
    cache, mom = mkv.alloc_cache(g, B + 1), mkv.alloc_moments(g)
    ws = mkv.alloc_workspace(mkv.mkv_compress_workspace_size(g, T, p))
    s = torch.zeros(1, H, T, device="cuda")
    s2 = torch.zeros_like(s)
    i1 = torch.zeros(1, H, B, dtype=torch.int32, device="cuda")
    mkv.mkv_compress(g, T, bf16(K), bf16(V), bf16(Q), p, cache, mom, ws, diag=(s, s2, i1))
    assert mkv.mkv_get_device_error(ws)[0] == 0
    got = dict(K=host(cache.K), V=host(cache.V), pos=host(cache.pos), len=host(cache.len), seen=host(cache.seen),
               n=host(mom.n), mu_k=host(mom.mu_k), mu_v=host(mom.mu_v), C=host(mom.C), s=host(s), s2=host(s2),
               i1=host(i1))
    for h in range(H):
        check_compress_unit(got, 0, h, K[0, h], V[0, h], Q[0, h], T, B, wl.window, wl.sink, True, 1, 1, 1e-6)
    out = torch.empty(1, H * G, G_.head_dim, device="cuda")
    wsd = mkv.alloc_workspace(mkv.mkv_decode_workspace_size(g, B + 1))
    mkv.mkv_decode_step(g, bf16(q[0]), bf16(kn[0]), bf16(vn[0]), cache, mom, mkv.mkv_decode_params(1, 1, 1e-6), out,
                        None, wsd)
    assert mkv.mkv_get_device_error(wsd)[0] == 0
    for h in range(H):
        R = got["pos"][0, h, :B]
        o, _, _, _ = O.decode_step(q[0, 0, h * G:(h + 1) * G], K[0, h][R], V[0, h][R],
                                   evicted_moments(K[0, h], V[0, h], R), kn[0, 0, h], vn[0, 0, h], True, 1, 1e-6)
        assert_output_close(host(out)[0, h * G:(h + 1) * G], o, f"decode after recovery, unit {h}")


@pytest.mark.parametrize("b,H,G,D,cap", [(1, 2, 2, 64, 300), (2, 8, 4, 128, 700), (40, 8, 2, 64, 96)])
def test_ticket_merge_against_oracle(b, H, G, D, cap):
    """The decode with its split-K partial states merged through global
    memory by the last CTA of each unit (atomic ticket)."""
    rng = np.random.default_rng(b * 100 + D)
    from test_zz_no_alloc import _case, _oracle_decode
    from gpu_util import f32, i32
    c = _case(rng, b, H, G, D, cap)
    g = mkv.geom(b, H, G, D)
    prev = mkv.mkv_debug_force_ticket_merge(1)
    try:
        for call in range(2):
            cache = mkv.Cache(bf16(c["K"]), bf16(c["V"]), i32(np.zeros((b, H, cap))), i32(c["lens"]),
                              i32(c["lens"]))
            mom = mkv.Moments(i32(c["n"]), f32(c["mu_k"]), f32(c["mu_v"]), f32(c["C"]))
            out = torch.full((b, H * G, D), float("nan"), device="cuda")
            lse = torch.full((b, H * G), float("nan"), device="cuda")
            ws = mkv.alloc_workspace(mkv.mkv_decode_workspace_size(g, cap))
            mkv.mkv_decode_step(g, bf16(c["q"]), bf16(c["kn"]), bf16(c["vn"]), cache, mom,
                                mkv.mkv_decode_params(1, 1, 1e-6), out, lse, ws)
            assert mkv.mkv_get_device_error(ws)[0] == 0
            want, want_lse = _oracle_decode(c["q"], c["K"], c["V"], c["lens"], c["n"], c["mu_k"], c["mu_v"], c["C"],
                                            c["kn"], c["vn"], G)
            assert_output_close(host(out), want, f"ticket merge call {call}")
            np.testing.assert_allclose(host(lse), want_lse, rtol=1e-4, atol=1e-4)
    finally:
        mkv.mkv_debug_force_ticket_merge(prev)
