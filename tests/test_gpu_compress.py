"""Prefill compression on the GPU against the fp64 oracle, through the C ABI:
window scores, the first- and second-stage retained sets (replayed on the
kernel's own scores, and equal to the oracle's wherever its boundary gap
exceeds 1e-5; below that the oracle continues from the kernel's choice), the
gathered cache, and the evicted-set moments (1e-4 relative).  Includes the tiny workload, ragged T, pooling,
mi off, T <= budget, 256 window rows, and the full Llama-3.1-8B one-layer
workload (T=8192, B=512, w=32); then the same with the budget shared by the
KV heads of a batch item (adaptive=1, Ada-KV allocation of Sec. 5.1) against
oracle.compress_adaptive, including a head count and prompt length whose
joint selection lists exceed the select kernel's shared-memory key cache."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2606_01563_gb300 import mkv
from paper_2606_01563_gb300.inputs import WORKLOADS, Generator, Geometry, Workload
from gpu_util import assert_moment_close, bf16, host
from parity import check_compress_item_adaptive, check_compress_unit, evicted_moments

pytestmark = pytest.mark.gpu


def run(wl, T=None, pool=1, mi=1, tau=1e-6, seed=0):
    gen = Generator(wl, seed=seed)
    K, V, Q = gen.prefill(T)
    g_ = wl.geom
    T = K.shape[2]
    B = wl.budget
    g = mkv.geom(g_.batch, g_.n_kv_heads, g_.group, g_.head_dim)
    p = mkv.mkv_compress_params(B, wl.window, wl.sink, wl.keep_window, pool, mi, 1, tau)
    cache = mkv.alloc_cache(g, B + 16)
    mom = mkv.alloc_moments(g)
    ws = mkv.alloc_workspace(mkv.mkv_compress_workspace_size(g, T, p))
    units = g_.batch * g_.n_kv_heads
    s = torch.zeros(g_.batch, g_.n_kv_heads, T, device="cuda")
    s2 = torch.zeros_like(s)
    i1 = torch.zeros(g_.batch, g_.n_kv_heads, B, dtype=torch.int32, device="cuda")
    mkv.mkv_compress(g, T, bf16(K), bf16(V), bf16(Q), p, cache, mom, ws, diag=(s, s2, i1))
    code, _ = mkv.mkv_get_device_error(ws)
    assert code == 0
    out = dict(K=host(cache.K), V=host(cache.V), pos=host(cache.pos), len=host(cache.len), seen=host(cache.seen),
               n=host(mom.n), mu_k=host(mom.mu_k), mu_v=host(mom.mu_v), C=host(mom.C), s=host(s), s2=host(s2),
               i1=host(i1))
    n_exact = 0
    for u in range(units):
        bi, h = divmod(u, g_.n_kv_heads)
        n_exact += check_compress_unit(out, bi, h, K[bi, h], V[bi, h], Q[bi, h], T, B, wl.window, wl.sink,
                                       bool(wl.keep_window), pool, mi, tau)
    out["_n_exact"] = n_exact
    return out


def test_tiny_workload():
    run(WORKLOADS["tiny_d64_t1k"])


def test_ragged_T_with_pooling():
    run(WORKLOADS["tiny_d64_t1k"], T=1000, pool=4, seed=3)


def test_mi_off_is_window_selection():
    run(WORKLOADS["tiny_d64_t1k"], mi=0, seed=4)


def test_budget_covers_prompt():
    wl = Workload("short", Geometry(1, 2, 2, 64), 100, 128, 16, "outlier")
    run(wl, seed=5)


def test_wide_window_256_rows():
    wl = Workload("w64", Geometry(1, 2, 4, 128), 4096, 128, 64, "mixture")
    run(wl, seed=6)


def test_batch_and_d128_ragged():
    wl = Workload("b2", Geometry(2, 2, 4, 128), 3001, 200, 32, "logscale")
    run(wl, seed=7)


def test_llama_layer_full_size():
    run(WORKLOADS["llama8b_layer_t8k"])


# ------------------------------------------------------- adaptive budget
def run_adaptive(wl, T=None, pool=1, mi=1, tau=1e-6, seed=0, cap_extra=0):
    """mkv_compress with adaptive=1 against oracle.compress_adaptive, per batch
    item: per-head scores, the joint first-stage list, score2, each head's
    retained set, length, rows and moments."""
    gen = Generator(wl, seed=seed)
    K, V, Q = gen.prefill(T)
    g_ = wl.geom
    T = K.shape[2]
    B, H = wl.budget, g_.n_kv_heads
    g = mkv.geom(g_.batch, H, g_.group, g_.head_dim)
    p = mkv.mkv_compress_params(B, wl.window, wl.sink, wl.keep_window, pool, mi, 1, tau, 1)
    prot = int(O.protected_mask(T, wl.window, wl.sink, bool(wl.keep_window)).sum())
    cap = min(T, H * (B - prot) + prot) + cap_extra
    cache = mkv.alloc_cache(g, cap)
    cache.K.normal_()  # stale rows: the padding the kernels read must be rewritten
    cache.V.normal_()
    mom = mkv.alloc_moments(g)
    ws = mkv.alloc_workspace(mkv.mkv_compress_workspace_size(g, T, p))
    s = torch.zeros(g_.batch, H, T, device="cuda")
    s2 = torch.zeros_like(s)
    i1 = torch.zeros(g_.batch, H * B, dtype=torch.int32, device="cuda")
    mkv.mkv_compress(g, T, bf16(K), bf16(V), bf16(Q), p, cache, mom, ws, diag=(s, s2, i1))
    code, _ = mkv.mkv_get_device_error(ws)
    assert code == 0
    out = dict(K=host(cache.K), V=host(cache.V), pos=host(cache.pos), len=host(cache.len), seen=host(cache.seen),
               n=host(mom.n), mu_k=host(mom.mu_k), mu_v=host(mom.mu_v), C=host(mom.C), s=host(s), s2=host(s2),
               i1=host(i1))
    n_exact = 0
    for bi in range(g_.batch):
        n_exact += check_compress_item_adaptive(out, bi, K[bi], V[bi], Q[bi], T, B, wl.window, wl.sink,
                                                bool(wl.keep_window), pool, mi, tau)
    return out, n_exact


def test_adaptive_tiny_workload():
    out, n = run_adaptive(WORKLOADS["tiny_d64_t1k"])
    assert n == 1


def test_adaptive_heads_keep_unequal_shares():
    wl = Workload("a4", Geometry(2, 4, 4, 128), 3001, 200, 32, "logscale")
    out, n = run_adaptive(wl, pool=4, seed=11, cap_extra=5)
    assert n >= 1
    assert len(np.unique(out["len"])) > 1  # the budget moved between heads


def test_adaptive_mi_off_mixture():
    wl = Workload("a8", Geometry(1, 8, 2, 64), 2048, 96, 16, "mixture")
    run_adaptive(wl, mi=0, seed=12)


def test_adaptive_budget_covers_prompt():
    wl = Workload("a-short", Geometry(1, 4, 2, 64), 100, 128, 16, "outlier")
    run_adaptive(wl, seed=13)


def test_adaptive_uncached_select_keys():
    # 8 heads x 60000 positions and a budget that leaves no per-head prefilter:
    # each select CTA's range of the joint list exceeds its shared-memory key cache
    wl = Workload("a-long", Geometry(1, 8, 1, 64), 60000, 4000, 16, "logscale")
    run_adaptive(wl, seed=14)


def test_adaptive_dense_joint_selection():
    # a unit may keep up to 1549 of its 2000 rows: the joint selection ranks every pair
    wl = Workload("a-dense", Geometry(1, 4, 2, 64), 2000, 400, 16, "outlier")
    out, n = run_adaptive(wl, seed=15, cap_extra=3)
    assert n == 1


def test_adaptive_llama_layer_full_size():
    run_adaptive(WORKLOADS["llama8b_layer_t8k"])


def test_adaptive_then_decode():
    """A decode step over the unequal per-head caches that the adaptive
    compression leaves, against the oracle's decode over its own sets."""
    from gpu_util import assert_output_close
    wl = Workload("a4d", Geometry(1, 4, 4, 128), 3001, 200, 32, "logscale")
    gen = Generator(wl, seed=21)
    K, V, Q = gen.prefill()
    G_, T, B = wl.geom, wl.T, wl.budget
    H, G, D = G_.n_kv_heads, G_.group, G_.head_dim
    g = mkv.geom(1, H, G, D)
    prot = 1 + wl.window
    cap = min(T, H * (B - prot) + prot) + 1
    cache, mom = mkv.alloc_cache(g, cap), mkv.alloc_moments(g)
    p = mkv.mkv_compress_params(B, wl.window, 1, 1, 1, 1, 1, 1e-6, 1)
    ws = mkv.alloc_workspace(mkv.mkv_compress_workspace_size(g, T, p))
    s = torch.zeros(1, H, T, device="cuda")
    s2 = torch.zeros_like(s)
    i1 = torch.zeros(1, H * B, dtype=torch.int32, device="cuda")
    mkv.mkv_compress(g, T, bf16(K), bf16(V), bf16(Q), p, cache, mom, ws, diag=(s, s2, i1))
    got = dict(K=host(cache.K), V=host(cache.V), pos=host(cache.pos), len=host(cache.len), seen=host(cache.seen),
               n=host(mom.n), mu_k=host(mom.mu_k), mu_v=host(mom.mu_v), C=host(mom.C), s=host(s), s2=host(s2),
               i1=host(i1))
    check_compress_item_adaptive(got, 0, K[0], V[0], Q[0], T, B, wl.window, 1, True, 1, 1, 1e-6)
    # the decode follows the compressed state the kernel left (the oracle's own
    # wherever its selections are exact, checked just above)
    R = [got["pos"][0, h, :got["len"][0, h]] for h in range(H)]
    rng = np.random.default_rng(5)
    q = (rng.standard_normal((1, H * G, D)) * 0.5).astype(np.float32)
    kn = rng.standard_normal((1, H, D)).astype(np.float32)
    vn = rng.standard_normal((1, H, D)).astype(np.float32)
    q, kn, vn = (host(bf16(x)) for x in (q, kn, vn))  # the bf16 values the kernel reads
    out = torch.empty(1, H * G, D, device="cuda")
    dws = mkv.alloc_workspace(mkv.mkv_decode_workspace_size(g, cap))
    mkv.mkv_decode_step(g, bf16(q), bf16(kn), bf16(vn), cache, mom, mkv.mkv_decode_params(1, 1, 1e-6), out, None,
                        dws)
    code, _ = mkv.mkv_get_device_error(dws)
    assert code == 0
    want = np.zeros((H * G, D))
    for h in range(H):
        idx = R[h]
        o, _, _, _ = O.decode_step(q[0, h * G:(h + 1) * G], K[0, h][idx], V[0, h][idx],
                                   evicted_moments(K[0, h], V[0, h], idx), kn[0, h], vn[0, h], True, 1, 1e-6)
        want[h * G:(h + 1) * G] = o
    assert_output_close(host(out)[0], want, "decode after adaptive compress")
    assert len(np.unique(host(cache.len))) > 1


def test_adaptive_head_with_no_retained_rows():
    """No protected rows and one free slot per head: head 0's window queries
    point at two of its keys, head 1's keys are near zero (flat attention), so
    the joint top 2 are both head 0's and head 1 keeps nothing (len 0; its
    moments cover all T rows)."""
    from paper_2606_01563_gb300.inputs import bf16_round
    rng = np.random.default_rng(41)
    T, d, g_, w = 256, 64, 2, 8
    K = np.empty((1, 2, T, d))
    K[0, 0] = rng.standard_normal((T, d))
    K[0, 1] = 0.01 * rng.standard_normal((T, d))
    V = rng.standard_normal((1, 2, T, d))
    Q = np.empty((1, 2, g_, w, d))
    for gi in range(g_):
        for i in range(w):
            tgt = K[0, 0, 10] if (gi + i) % 2 == 0 else K[0, 0, 200]
            Q[0, 0, gi, i] = 3.0 * tgt
    Q[0, 1] = rng.standard_normal((g_, w, d))
    K, V, Q = bf16_round(K), bf16_round(V), bf16_round(Q)
    g = mkv.geom(1, 2, g_, d)
    p = mkv.mkv_compress_params(1, w, 0, 0, 1, 1, 1, 1e-6, 1)
    cache, mom = mkv.alloc_cache(g, 2), mkv.alloc_moments(g)
    ws = mkv.alloc_workspace(mkv.mkv_compress_workspace_size(g, T, p))
    mkv.mkv_compress(g, T, bf16(K), bf16(V), bf16(Q), p, cache, mom, ws)
    assert mkv.mkv_get_device_error(ws)[0] == 0
    ref = O.compress_adaptive(K[0], V[0], Q[0], 1, w, 0, False, 1, True, 1e-6)
    assert [len(r) for r in ref.idx] == [2, 0]
    np.testing.assert_array_equal(host(cache.len)[0], [2, 0])
    np.testing.assert_array_equal(host(cache.pos)[0, 0], ref.idx[0])
    for h in range(2):
        m = ref.moments[h]
        assert host(mom.n)[0, h] == m.n
        assert_moment_close(host(mom.mu_k)[0, h], m.mu_k, "mu_k")
        assert_moment_close(host(mom.mu_v)[0, h], m.mu_v, "mu_v")
        assert_moment_close(host(mom.C)[0, h], m.C, "C")
