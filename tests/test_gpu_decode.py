"""Decode step (Algorithm 1 Phase 2) on the GPU against the fp64 oracle,
through the C ABI.  Covers head dims 64/128, groups 1/2/4/8, ragged lengths
that cross tile and split boundaries, append on/off, correction on/off,
order 0/1, the clamp, empty retained sets, per-unit moment counts including
n = 0, device-detected errors, and the full-size decode sweep cells."""
import math

import numpy as np
import pytest
import torch

import oracle as O
from paper_2606_01563_gb300 import mkv
from paper_2606_01563_gb300.inputs import bf16_round
from gpu_util import assert_output_close, bf16, f32, host, i32

pytestmark = pytest.mark.gpu


def make_state(rng, b, H, G, D, lens, cap, n_list, key_scale=1.0):
    units = b * H
    K = bf16_round(key_scale * rng.standard_normal((b, H, cap, D)))
    V = bf16_round(rng.standard_normal((b, H, cap, D)))
    n = np.array(n_list, np.int32).reshape(b, H)
    mu_k = (0.3 * rng.standard_normal((b, H, D))).astype(np.float32)
    mu_v = (0.3 * rng.standard_normal((b, H, D))).astype(np.float32)
    C = (0.05 * rng.standard_normal((b, H, D, D))).astype(np.float32)
    lens = np.array(lens, np.int32).reshape(b, H)
    q = bf16_round(2.0 * rng.standard_normal((b, H * G, D)))
    kn = bf16_round(key_scale * rng.standard_normal((b, H, D)))
    vn = bf16_round(rng.standard_normal((b, H, D)))
    return dict(K=K, V=V, n=n, mu_k=mu_k, mu_v=mu_v, C=C, lens=lens, q=q, kn=kn, vn=vn, cap=cap)


def run_gpu(st, b, H, G, D, new, correction, order, tau):
    g = mkv.geom(b, H, G, D)
    cache = mkv.Cache(bf16(st["K"]), bf16(st["V"]),
                      i32(np.broadcast_to(np.arange(st["cap"]), (b, H, st["cap"]))),
                      i32(st["lens"]), i32(st["lens"] + 1000))
    mom = mkv.Moments(i32(st["n"]), f32(st["mu_k"]), f32(st["mu_v"]), f32(st["C"]))
    out = torch.empty(b, H * G, D, device="cuda")
    lse = torch.empty(b, H * G, device="cuda")
    ws = mkv.alloc_workspace(mkv.mkv_decode_workspace_size(g, st["cap"]))
    p = mkv.mkv_decode_params(correction, order, tau)
    kn = bf16(st["kn"]) if new else None
    vn = bf16(st["vn"]) if new else None
    mkv.mkv_decode_step(g, bf16(st["q"]), kn, vn, cache, mom, p, out, lse, ws)
    code, info = mkv.mkv_get_device_error(ws)
    return host(out), host(lse), cache, code, info, ws


def run_oracle(st, b, H, G, D, new, correction, order, tau):
    out = np.zeros((b, H * G, D))
    lse = np.zeros((b, H * G))
    for bi in range(b):
        for h in range(H):
            L = st["lens"][bi, h]
            m = O.Moments(int(st["n"][bi, h]), st["mu_k"][bi, h], st["mu_v"][bi, h], st["C"][bi, h])
            o, l, _, _ = O.decode_step(st["q"][bi, h * G:(h + 1) * G], st["K"][bi, h, :L], st["V"][bi, h, :L], m,
                                       st["kn"][bi, h] if new else None, st["vn"][bi, h] if new else None,
                                       bool(correction), order, tau)
            out[bi, h * G:(h + 1) * G] = o
            lse[bi, h * G:(h + 1) * G] = l
    return out, lse


CASES = [
    # b, H, G, D, lens, cap, n_list
    (1, 2, 2, 64, [100, 37], 160, [50, 3]),
    (2, 8, 4, 128, None, 640, None),
    (1, 4, 8, 128, [513, 1, 32, 33], 600, [10, 0, 1, 1000]),
    (3, 2, 1, 64, [31, 64, 65, 200, 7, 129], 256, [0, 5, 9, 100, 2, 40]),
    # 320 units: one split per unit, so each CTA computes all 64 moment rows
    (40, 8, 2, 64, None, 96, None),
]


@pytest.mark.parametrize("case", range(len(CASES)))
@pytest.mark.parametrize("new", [False, True])
@pytest.mark.parametrize("correction,order", [(1, 1), (1, 0), (0, 1)])
def test_decode_matches_oracle(case, new, correction, order):
    b, H, G, D, lens, cap, n_list = CASES[case]
    rng = np.random.default_rng(100 + case)
    if lens is None:
        lens = rng.integers(1, cap - 1, b * H)
    if n_list is None:
        n_list = rng.integers(0, 5000, b * H)
    st = make_state(rng, b, H, G, D, lens, cap, n_list)
    out, lse, cache, code, _, _ = run_gpu(st, b, H, G, D, new, correction, order, 1e-6)
    ref, ref_lse = run_oracle(st, b, H, G, D, new, correction, order, 1e-6)
    assert code == 0
    assert_output_close(out, ref, "decode out")
    np.testing.assert_allclose(lse, ref_lse, rtol=0, atol=1e-4 * np.maximum(1, np.abs(ref_lse)).max())
    lens_after = host(cache.len)
    np.testing.assert_array_equal(lens_after, st["lens"] + (1 if new else 0))
    if new:
        Kc = host(cache.K)
        for bi in range(b):
            for h in range(H):
                L = st["lens"][bi, h]
                np.testing.assert_array_equal(Kc[bi, h, L], st["kn"][bi, h])
                assert host(cache.pos)[bi, h, L] == st["lens"][bi, h] + 1000
        np.testing.assert_array_equal(host(cache.seen), st["lens"] + 1001)


def test_clamp_everything_reduces_to_order0():
    rng = np.random.default_rng(7)
    st = make_state(rng, 1, 2, 4, 128, [90, 300], 320, [20, 400])
    out_big, _, _, code, _, _ = run_gpu(st, 1, 2, 4, 128, False, 1, 1, 1e9)
    ref, _ = run_oracle(st, 1, 2, 4, 128, False, 1, 0, 0.0)
    assert code == 0
    assert_output_close(out_big, ref, "clamp-all")


def test_empty_retained_set():
    rng = np.random.default_rng(8)
    st = make_state(rng, 1, 2, 2, 64, [0, 0], 64, [7, 0])
    out, lse, _, code, info, _ = run_gpu(st, 1, 2, 2, 64, False, 1, 1, 0.0)
    # unit 0: no rows, moments present -> f_hat_E; unit 1: nothing at all -> error
    m = O.Moments(7, st["mu_k"][0, 0], st["mu_v"][0, 0], st["C"][0, 0])
    for h in range(2):
        assert_output_close(out[0, h][None], O.fhat_E(st["q"][0, h], m)[None], "f_hat_E only")
    assert code == 1 and info == 1
    # the same workspace works again after the error was read and cleared
    st["lens"][:] = 5
    out, _, _, code, _, _ = run_gpu(st, 1, 2, 2, 64, False, 1, 1, 0.0)
    assert code == 0


def test_append_past_capacity_is_reported():
    rng = np.random.default_rng(9)
    st = make_state(rng, 1, 2, 2, 64, [64, 10], 64, [3, 3])
    out, _, cache, code, info, _ = run_gpu(st, 1, 2, 2, 64, True, 1, 1, 0.0)
    assert code == 3 and info == 0
    np.testing.assert_array_equal(host(cache.len), [[64, 11]])
    ref, _ = run_oracle(st, 1, 2, 2, 64, True, 1, 1, 0.0)
    assert_output_close(out, ref, "attends over the new token anyway")


def test_workspace_reused_across_steps():
    """The split-K ticket counters reset themselves: 5 appends in a row."""
    rng = np.random.default_rng(10)
    b, H, G, D, cap = 1, 8, 4, 128, 600
    st = make_state(rng, b, H, G, D, [500] * 8, cap, [4000] * 8)
    g = mkv.geom(b, H, G, D)
    cache = mkv.Cache(bf16(st["K"]), bf16(st["V"]), i32(np.zeros((b, H, cap))), i32(st["lens"]),
                      i32(st["lens"]))
    mom = mkv.Moments(i32(st["n"]), f32(st["mu_k"]), f32(st["mu_v"]), f32(st["C"]))
    ws = mkv.alloc_workspace(mkv.mkv_decode_workspace_size(g, cap))
    p = mkv.mkv_decode_params(1, 1, 1e-6)
    Kh, Vh = st["K"].copy(), st["V"].copy()
    for step in range(5):
        q = bf16_round(2.0 * rng.standard_normal((b, H * G, D)))
        kn = bf16_round(rng.standard_normal((b, H, D)))
        vn = bf16_round(rng.standard_normal((b, H, D)))
        out = torch.empty(b, H * G, D, device="cuda")
        mkv.mkv_decode_step(g, bf16(q), bf16(kn), bf16(vn), cache, mom, p, out, None, ws)
        L = 500 + step
        for h in range(H):
            Kh[0, h, L], Vh[0, h, L] = kn[0, h], vn[0, h]
            m = O.Moments(4000, st["mu_k"][0, h], st["mu_v"][0, h], st["C"][0, h])
            ref, _, _, _ = O.decode_step(q[0, h * G:(h + 1) * G], Kh[0, h, :L + 1], Vh[0, h, :L + 1], m,
                                         tau=1e-6)
            assert_output_close(host(out)[0, h * G:(h + 1) * G], ref, f"step {step}")
    assert mkv.mkv_get_device_error(ws)[0] == 0


@pytest.mark.parametrize("batch", [1, 8, 32, 64])
@pytest.mark.parametrize("budget", [256, 1024, 4096])
def test_decode_sweep_full_size(batch, budget):
    """Llama-3.1-8B geometry decode sweep cells (32 query heads, 8 KV heads,
    d=128, dense fp32 C) at full size, every output checked."""
    rng = np.random.default_rng(batch * 7 + budget)
    b, H, G, D = batch, 8, 4, 128
    cap = budget + 64
    st = make_state(rng, b, H, G, D, [budget] * (b * H), cap, [8192 - budget] * (b * H))
    out, lse, _, code, _, _ = run_gpu(st, b, H, G, D, True, 1, 1, 1e-6)
    ref, ref_lse = run_oracle(st, b, H, G, D, True, 1, 1, 1e-6)
    assert code == 0
    assert_output_close(out, ref, "sweep")
    np.testing.assert_allclose(lse, ref_lse, rtol=0, atol=1e-3)


@pytest.mark.parametrize("case", [1, 4])
@pytest.mark.parametrize("order", [1, 0])
def test_decode_bf16_moment_storage(case, order):
    """16-bit moment storage: mkv_moments_pack_bf16 rounds C to bf16 exactly as
    torch does, and decode reading that copy matches the oracle run on the
    bf16-rounded C (order 0 ignores C)."""
    b, H, G, D, lens, cap, n_list = CASES[case]
    rng = np.random.default_rng(300 + case)
    if lens is None:
        lens = rng.integers(1, cap - 1, b * H)
    if n_list is None:
        n_list = rng.integers(0, 5000, b * H)
    st = make_state(rng, b, H, G, D, lens, cap, n_list)
    g = mkv.geom(b, H, G, D)
    mom = mkv.Moments(i32(st["n"]), f32(st["mu_k"]), f32(st["mu_v"]), f32(st["C"]))
    C16 = torch.empty(b, H, D, D, dtype=torch.bfloat16, device="cuda")
    mkv.mkv_moments_pack_bf16(g, mom, C16)
    ref16 = torch.from_numpy(st["C"]).to(torch.bfloat16)
    assert torch.equal(C16.cpu().view(torch.int16), ref16.view(torch.int16))
    cache = mkv.Cache(bf16(st["K"]), bf16(st["V"]),
                      i32(np.broadcast_to(np.arange(st["cap"]), (b, H, st["cap"]))),
                      i32(st["lens"]), i32(st["lens"] + 1000))
    out = torch.empty(b, H * G, D, device="cuda")
    lse = torch.empty(b, H * G, device="cuda")
    ws = mkv.alloc_workspace(mkv.mkv_decode_workspace_size(g, st["cap"]))
    p = mkv.mkv_decode_params(1, order, 1e-6, C16.data_ptr())
    mkv.mkv_decode_step(g, bf16(st["q"]), bf16(st["kn"]), bf16(st["vn"]), cache, mom, p, out, lse, ws)
    code, _ = mkv.mkv_get_device_error(ws)
    assert code == 0
    st16 = dict(st, C=ref16.float().numpy())
    ref, ref_lse = run_oracle(st16, b, H, G, D, True, 1, order, 1e-6)
    assert_output_close(host(out), ref, "decode out (bf16 C)")
    np.testing.assert_allclose(host(lse), ref_lse, rtol=0, atol=1e-4 * np.maximum(1, np.abs(ref_lse)).max())
