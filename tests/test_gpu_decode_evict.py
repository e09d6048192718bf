"""One decoding step of Algorithm 1 (append, Phase 1 down to the budget,
Phase 2) on the GPU against the fp64 oracle, through the C ABI: the oracle
follows the kernel's evictions (each the argmin of Algorithm 1's scores under
the state reached, or at a near tie one of the near-minimal rows), then
decodes over the state reached; the corrected output and its log-normaliser
(2e-3 of the output's max-abs), the surviving rows (exact), and the updated
moments (1e-4 relative).  Covers the register eviction kernel and the
larger-cache eviction kernels ahead of the decode kernel, steps with nothing
to evict, eviction down to an empty cache, and several continuous steps."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2606_01563_gb300 import mkv
from paper_2606_01563_gb300.inputs import bf16_round
from gpu_util import assert_output_close, bf16, f32, host, i32
from parity import check_evicted_unit
from test_gpu_evict import setup

pytestmark = pytest.mark.gpu


def run_steps(st, b, H, G, D, budget, steps=1, correction=1, order=1, tau=1e-6, seed=0, evict_state=False):
    """`steps` calls of mkv_decode_evict_step, each with fresh queries and a
    new token, against the oracle carrying its own state.  evict_state: the
    cache keeps y_j = S_tilde k_j across calls (mkv_cache.y, y_len)."""
    rng = np.random.default_rng(seed)
    g = mkv.geom(b, H, G, D)
    cap = st["cap"]
    pos0 = np.broadcast_to(np.arange(cap, dtype=np.int32) * 3, (b, H, cap)).copy()
    seen0 = 10 ** 6
    cache = mkv.Cache(bf16(st["K"]), bf16(st["V"]), i32(pos0), i32(st["lens"]), i32(np.full((b, H), seen0)))
    if evict_state:
        cache.y = torch.zeros(b, H, cap, D, device="cuda")
        cache.y_len = torch.zeros(b, H, dtype=torch.int32, device="cuda")
    mom = mkv.Moments(i32(st["n"]), f32(st["mu_k"]), f32(st["mu_v"]), f32(st["C"]))
    ws = mkv.alloc_workspace(mkv.mkv_decode_evict_workspace_size(g, cap))
    p = mkv.mkv_decode_params(correction, order, tau)
    ref = {}
    for bi in range(b):
        for h in range(H):
            L = st["lens"][bi, h]
            ref[bi, h] = dict(K=st["K"][bi, h, :L], V=st["V"][bi, h, :L], pos=pos0[bi, h, :L],
                              m=O.Moments(int(st["n"][bi, h]), st["mu_k"][bi, h], st["mu_v"][bi, h], st["C"][bi, h]))
    for step in range(steps):
        if step > 0:
            st = dict(st, q=bf16_round(2.0 * rng.standard_normal((b, H * G, D))),
                      kn=bf16_round(1.5 * rng.standard_normal((b, H, D))),
                      vn=bf16_round(rng.standard_normal((b, H, D))))
        out = torch.full((b, H * G, D), float("nan"), device="cuda")
        lse = torch.full((b, H * G), float("nan"), device="cuda")
        mkv.mkv_decode_evict_step(g, bf16(st["q"]), bf16(st["kn"]), bf16(st["vn"]), budget, cache, mom, p, out, lse,
                                  ws)
        code, info = mkv.mkv_get_device_error(ws)
        assert code == 0, (code, info)
        got = dict(out=host(out), lse=host(lse), K=host(cache.K), V=host(cache.V), pos=host(cache.pos),
                   len=host(cache.len), seen=host(cache.seen), n=host(mom.n), mu_k=host(mom.mu_k),
                   mu_v=host(mom.mu_v), C=host(mom.C))
        for (bi, h), s in ref.items():
            q = st["q"][bi, h * G:(h + 1) * G]
            K = np.vstack([s["K"], st["kn"][bi, h][None]])
            V = np.vstack([s["V"], st["vn"][bi, h][None]])
            pos = np.append(s["pos"], seen0 + step)
            # Phase 1: the oracle follows the kernel's evictions (exact argmin,
            # or one of the near-minimal rows at a near tie)
            f = check_evicted_unit(got, bi, h, q, K, V, pos, s["m"], budget, tau)
            assert got["seen"][bi, h] == seen0 + step + 1
            # Phase 2 over the state reached
            o, l, _, _ = O.decode_step(q, f.K, f.V, f.moments, None, None, bool(correction), order, tau)
            assert_output_close(got["out"][bi, h * G:(h + 1) * G], o, f"out step {step} unit {(bi, h)}")
            np.testing.assert_allclose(got["lse"][bi, h * G:(h + 1) * G], l, rtol=1e-4, atol=1e-4)
            s.update(K=f.K, V=f.V, pos=f.pos, m=f.moments)
        if evict_state:
            check_y_rows(cache, mom)
    return got


def check_y_rows(cache, mom):
    """The cache's current y rows equal S_tilde k_j = n C k_j of the kernel's
    own moments and rows (1e-4 of the largest, per unit)."""
    y, y_len, K = host(cache.y), host(cache.y_len), host(cache.K).astype(np.float64)
    n, C = host(mom.n), host(mom.C).astype(np.float64)
    for bi in range(y.shape[0]):
        for h in range(y.shape[1]):
            L = int(y_len[bi, h])
            assert 0 <= L <= int(host(cache.len)[bi, h])
            if L == 0 or n[bi, h] == 0:
                continue
            want = K[bi, h, :L] @ (n[bi, h] * C[bi, h]).T
            err = np.abs(y[bi, h, :L] - want).max()
            assert err <= 1e-4 * np.abs(want).max(), (bi, h, err, np.abs(want).max())


def test_tiny_several_evictions_in_one_step():
    rng = np.random.default_rng(31)
    st = setup(rng, 1, 2, 2, 64, [40, 33], 48, [0, 25])
    run_steps(st, 1, 2, 2, 64, 24)


@pytest.mark.parametrize("correction,order", [(1, 1), (1, 0), (0, 1)])
def test_llama_continuous_one_eviction_per_step(correction, order):
    """Cache at the budget (512 of 576 rows): every step appends and evicts one."""
    rng = np.random.default_rng(32)
    st = setup(rng, 1, 8, 4, 128, [512] * 8, 576, [3000] * 4 + [0] * 4)
    run_steps(st, 1, 8, 4, 128, 512, steps=3, correction=correction, order=order, seed=5)


def test_below_budget_nothing_evicted():
    rng = np.random.default_rng(33)
    st = setup(rng, 2, 2, 2, 64, [10, 3, 0, 7], 16, [0, 1, 2, 3])
    run_steps(st, 2, 2, 2, 64, 12)


def test_evict_to_empty_cache_gives_moment_term():
    rng = np.random.default_rng(34)
    st = setup(rng, 1, 2, 4, 64, [5, 2], 8, [7, 1])
    run_steps(st, 1, 2, 4, 64, 0)


def test_large_cache_eviction_kernel():
    """Capacity 1300 (> 8 x 144 rows): the shared-memory cluster eviction kernel."""
    rng = np.random.default_rng(35)
    st = setup(rng, 1, 2, 2, 128, [1200, 1100], 1300, [500, 0])
    run_steps(st, 1, 2, 2, 128, 1150, steps=2, seed=6)


def test_group_8_d64_batch():
    rng = np.random.default_rng(36)
    st = setup(rng, 2, 2, 8, 64, [100, 64, 65, 99], 128, [10, 0, 200, 3])
    run_steps(st, 2, 2, 8, 64, 64, steps=2, seed=7)


@pytest.mark.parametrize("G", [4, 1])
def test_continuous_with_eviction_state(G):
    """Continuous eviction with y_j = S_tilde k_j kept in the cache across
    calls: the first call fills it, the next ones compute it only for the
    appended token; every step against the oracle, and the kept y rows
    against n C k_j of the kernel's own moments."""
    rng = np.random.default_rng(40 + G)
    st = setup(rng, 1, 8, G, 128, [512] * 8, 576, [3000] * 6 + [0] * 2)
    run_steps(st, 1, 8, G, 128, 512, steps=4, seed=8, evict_state=True)


def test_eviction_state_several_evictions_per_step_d64():
    rng = np.random.default_rng(42)
    st = setup(rng, 2, 2, 2, 64, [40, 33, 45, 20], 48, [0, 25, 3, 7])
    run_steps(st, 2, 2, 2, 64, 24, steps=3, seed=9, evict_state=True)
