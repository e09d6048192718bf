"""Prefill compression at the full long-context sizes the benchmark times,
through the C ABI, checked on sampled units against the fp64 oracle:
  - Qwen3-4B geometry, batch 4, T = 32768, budget 1024, window 32 (per-unit
    budget, and the budget shared by the KV heads of a batch item);
  - Llama-3.1-8B geometry, T = 131072, budget 128, window 64 (Gaussian-mixture
    keys).
The inputs are the benchmark's (same workloads, same seed).  The oracle
recomputes a sampled unit (or batch item) from its own prompt slice.

What is compared:
  - window scores and score2 within tolerance;
  - each selection replayed on the kernel's own fp32 scores: the radix select
    must return exactly the top k of the values it ranked, lower position
    first on ties;
  - the selection equal to the oracle's wherever the oracle's boundary gap
    exceeds 1e-5 (relative);
  - otherwise, a near tie decides the boundary and either side of it is a
    correct answer.  Then the oracle continues from the kernel's choice
    (score2 under the kernel's stage-1 set, moments of the kernel's evicted
    set), so the rest is still compared element by element;
  - gathered rows bit-exact, moments within 1e-4 relative.
"""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2606_01563_gb300 import mkv
from paper_2606_01563_gb300.inputs import WORKLOADS, Generator
from gpu_util import GAP_EXACT, assert_moment_close, bf16, host

pytestmark = pytest.mark.gpu

SEED = 11  # the benchmark's long-context compress inputs
TAU = 1e-6


def _prefill(name):
    wl = WORKLOADS[name]
    K, V, Q = Generator(wl, seed=SEED).prefill()
    return wl, K, V, Q


def _compress_gpu(wl, K, V, Q, adaptive):
    G = wl.geom
    H, T, B = G.n_kv_heads, wl.T, wl.budget
    g = mkv.geom(G.batch, H, G.group, G.head_dim)
    p = mkv.mkv_compress_params(B, wl.window, wl.sink, wl.keep_window, 1, 1, 1, TAU, adaptive)
    prot = wl.sink + (wl.window if wl.keep_window else 0)
    cap = min(T, H * (B - prot) + prot) if adaptive else B + 64  # as the benchmark allocates
    cache, mom = mkv.alloc_cache(g, cap), mkv.alloc_moments(g)
    ws = mkv.alloc_workspace(mkv.mkv_compress_workspace_size(g, T, p))
    s = torch.zeros(G.batch, H, T, device="cuda")
    s2 = torch.zeros_like(s)
    shape = (G.batch, H * B) if adaptive else (G.batch, H, B)
    i1 = torch.zeros(shape, dtype=torch.int32, device="cuda")
    mkv.mkv_compress(g, T, bf16(K), bf16(V), bf16(Q), p, cache, mom, ws, diag=(s, s2, i1))
    code, _ = mkv.mkv_get_device_error(ws)
    assert code == 0
    out = dict(K=host(cache.K), V=host(cache.V), pos=host(cache.pos), len=host(cache.len), seen=host(cache.seen),
               n=host(mom.n), mu_k=host(mom.mu_k), mu_v=host(mom.mu_v), C=host(mom.C),
               s=host(s).astype(np.float64), s2=host(s2).astype(np.float64),
               i1=host(i1))
    del cache, mom, ws, s, s2, i1
    torch.cuda.empty_cache()
    return out


def _score2_under(K, V, s, R0):
    """Oracle score2 (Eq. residual under the moments of all \\ R0, times s)
    for a given stage-1 set R0."""
    keep0 = np.zeros(K.shape[0], bool)
    keep0[R0] = True
    r = O.residual(K, V, O.moments_of(K[~keep0], V[~keep0]), TAU)
    return s * np.sqrt((r * r).sum(axis=1))


def _check_rows_and_moments(out, bi, h, K, V, R, m):
    n_r = len(R)
    np.testing.assert_array_equal(out["K"][bi, h, :n_r], K[R])
    np.testing.assert_array_equal(out["V"][bi, h, :n_r], V[R])
    assert out["n"][bi, h] == m.n
    if m.n:
        assert_moment_close(out["mu_k"][bi, h], m.mu_k, "mu_k")
        assert_moment_close(out["mu_v"][bi, h], m.mu_v, "mu_v")
        assert_moment_close(out["C"][bi, h], m.C, "C")
    else:
        assert not out["C"][bi, h].any()


def _evicted_moments(K, V, R):
    keep = np.zeros(K.shape[0], bool)
    keep[R] = True
    return O.moments_of(K[~keep], V[~keep])


def check_unit(out, wl, bi, h, K, V, Q):
    """One (batch, KV head) unit of a per-unit-budget compress."""
    T, B = wl.T, wl.budget
    ref = O.compress(K, V, Q, B, wl.window, wl.sink, bool(wl.keep_window), 1, True, TAU)
    prot = O.protected_mask(T, wl.window, wl.sink, bool(wl.keep_window))
    free = ~prot
    k = B - int(prot.sum())
    s_g, s2_g = out["s"][bi, h], out["s2"][bi, h]
    np.testing.assert_allclose(s_g, ref.scores, rtol=2e-5, atol=2e-6 * ref.scores.max())
    # stage 1: the kernel's choice is the exact top k of its own scores
    R0 = out["i1"][bi, h]
    np.testing.assert_array_equal(R0, O.select_topk(s_g, k, prot)[0])
    if ref.gap1 > GAP_EXACT:
        np.testing.assert_array_equal(R0, ref.idx_stage1)
        score2 = ref.score2
    else:
        score2 = _score2_under(K, V, ref.scores, R0)
    np.testing.assert_allclose(s2_g[free], score2[free], rtol=1e-4, atol=1e-5 * score2[free].max())
    # stage 2 into the cache
    assert out["len"][bi, h] == B and out["seen"][bi, h] == T
    R = out["pos"][bi, h, :B]
    np.testing.assert_array_equal(R, O.select_topk(s2_g, k, prot)[0])
    if ref.gap1 > GAP_EXACT and ref.gap2 > GAP_EXACT:
        np.testing.assert_array_equal(R, ref.idx)
        m = ref.moments
    else:
        m = _evicted_moments(K, V, R)
    _check_rows_and_moments(out, bi, h, K, V, R, m)
    return ref.gap1 > GAP_EXACT and ref.gap2 > GAP_EXACT


def check_item_adaptive(out, wl, bi, K, V, Q):
    """The KV heads of batch item bi, budget shared across them (K, V: [H, T, d])."""
    T, B = wl.T, wl.budget
    H = K.shape[0]
    ref = O.compress_adaptive(K, V, Q, B, wl.window, wl.sink, bool(wl.keep_window), 1, True, TAU)
    prot = np.stack([O.protected_mask(T, wl.window, wl.sink, bool(wl.keep_window))] * H)
    k = H * B - int(prot.sum())
    s_g, s2_g = out["s"][bi], out["s2"][bi]
    for h in range(H):
        np.testing.assert_allclose(s_g[h], ref.scores[h], rtol=2e-5, atol=2e-6 * ref.scores[h].max())

    def flat(lists):
        return np.concatenate([h * T + r for h, r in enumerate(lists)])

    R0 = O.select_topk_joint(s_g, k, prot)[0]
    np.testing.assert_array_equal(out["i1"][bi], flat(R0))
    if ref.gap1 > GAP_EXACT:
        np.testing.assert_array_equal(flat(R0), flat(ref.idx_stage1))
        score2 = ref.score2
    else:
        score2 = np.stack([_score2_under(K[h], V[h], ref.scores[h], R0[h]) for h in range(H)])
    for h in range(H):
        free = ~prot[h]
        np.testing.assert_allclose(s2_g[h][free], score2[h][free], rtol=1e-4,
                                   atol=1e-5 * score2[h][free].max())
    assert (out["seen"][bi] == T).all() and out["len"][bi].sum() == H * B
    R = [out["pos"][bi, h, :out["len"][bi, h]] for h in range(H)]
    want = O.select_topk_joint(s2_g, k, prot)[0]
    np.testing.assert_array_equal(flat(R), flat(want))
    exact = ref.gap1 > GAP_EXACT and ref.gap2 > GAP_EXACT
    if exact:
        np.testing.assert_array_equal(flat(R), flat(ref.idx))
    for h in range(H):
        m = ref.moments[h] if exact else _evicted_moments(K[h], V[h], R[h])
        _check_rows_and_moments(out, bi, h, K[h], V[h], R[h], m)
    return exact


@pytest.fixture(scope="module")
def qwen32k():
    return _prefill("qwen4b_t32k")


def test_compress_qwen4b_t32k_batch4_sampled_units(qwen32k):
    wl, K, V, Q = qwen32k
    out = _compress_gpu(wl, K, V, Q, adaptive=0)
    for bi, h in ((0, 0), (1, 5), (3, 7)):
        check_unit(out, wl, bi, h, K[bi, h], V[bi, h], Q[bi, h])


def test_compress_qwen4b_t32k_adaptive_sampled_item(qwen32k):
    wl, K, V, Q = qwen32k
    out = _compress_gpu(wl, K, V, Q, adaptive=1)
    check_item_adaptive(out, wl, 2, K[2], V[2], Q[2])


def test_compress_llama8b_t128k_sampled_units():
    wl, K, V, Q = _prefill("llama8b_t128k")
    out = _compress_gpu(wl, K, V, Q, adaptive=0)
    for h in (0, 7):
        check_unit(out, wl, 0, h, K[0, h], V[0, h], Q[0, h])
