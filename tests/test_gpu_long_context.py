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

from paper_2606_01563_gb300 import mkv
from paper_2606_01563_gb300.inputs import WORKLOADS, Generator
from gpu_util import bf16, host
from parity import check_compress_item_adaptive, check_compress_unit

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


def check_unit(out, wl, bi, h, K, V, Q):
    return check_compress_unit(out, bi, h, K, V, Q, wl.T, wl.budget, wl.window, wl.sink, bool(wl.keep_window), 1, 1,
                               TAU)


def check_item_adaptive(out, wl, bi, K, V, Q):
    return check_compress_item_adaptive(out, bi, K, V, Q, wl.T, wl.budget, wl.window, wl.sink,
                                        bool(wl.keep_window), 1, 1, TAU)


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
