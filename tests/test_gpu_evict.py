"""Moment-informed eviction (Algorithm 1 append + Phase 1) on the GPU against
the fp64 oracle, through the C ABI: every eviction is the oracle's argmin
under the state reached so far, or at a near tie (argmin gap within 1e-5)
one of the near-minimal rows, and the oracle follows the kernel's choice;
the surviving rows in order and the updated moments (1e-4 relative)."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2606_01563_gb300 import mkv
from paper_2606_01563_gb300.inputs import bf16_round
from gpu_util import bf16, f32, host, i32
from parity import check_evicted_unit

pytestmark = pytest.mark.gpu


def setup(rng, b, H, G, D, lens, cap, n_evicted0):
    """Cache rows and moments that come from a real evicted set of size n_evicted0."""
    st = {"K": bf16_round(1.5 * rng.standard_normal((b, H, cap, D))),
          "V": bf16_round(rng.standard_normal((b, H, cap, D))),
          "lens": np.array(lens, np.int32).reshape(b, H),
          "q": bf16_round(2.0 * rng.standard_normal((b, H * G, D))),
          "kn": bf16_round(1.5 * rng.standard_normal((b, H, D))),
          "vn": bf16_round(rng.standard_normal((b, H, D)))}
    n = np.zeros((b, H), np.int32)
    mk = np.zeros((b, H, D), np.float32)
    mv = np.zeros((b, H, D), np.float32)
    C = np.zeros((b, H, D, D), np.float32)
    for bi in range(b):
        for h in range(H):
            ne = n_evicted0[bi * H + h]
            if ne:
                m = O.moments_of(bf16_round(1.5 * rng.standard_normal((ne, D))),
                                 bf16_round(rng.standard_normal((ne, D))))
                n[bi, h], mk[bi, h], mv[bi, h], C[bi, h] = m.n, m.mu_k, m.mu_v, m.C
    st.update(n=n, mu_k=mk, mu_v=mv, C=C, cap=cap)
    return st


def run_case(st, b, H, G, D, budget, new, tau=1e-6):
    g = mkv.geom(b, H, G, D)
    cap = st["cap"]
    pos0 = np.broadcast_to(np.arange(cap, dtype=np.int32) * 3, (b, H, cap)).copy()
    cache = mkv.Cache(bf16(st["K"]), bf16(st["V"]), i32(pos0), i32(st["lens"]), i32(np.full((b, H), 10 ** 6)))
    mom = mkv.Moments(i32(st["n"]), f32(st["mu_k"]), f32(st["mu_v"]), f32(st["C"]))
    ws = mkv.alloc_workspace(mkv.mkv_evict_workspace_size(g, cap))
    mkv.mkv_evict_append(g, bf16(st["q"]), bf16(st["kn"]) if new else None, bf16(st["vn"]) if new else None,
                         budget, cache, mom, tau, ws)
    code, info = mkv.mkv_get_device_error(ws)
    gpu = dict(K=host(cache.K), V=host(cache.V), pos=host(cache.pos), len=host(cache.len), seen=host(cache.seen),
               n=host(mom.n), mu_k=host(mom.mu_k), mu_v=host(mom.mu_v), C=host(mom.C), code=code, info=info,
               pos0=pos0, G=G, budget=budget, new=new, tau=tau)
    return gpu


def unit_state(st, pos0, bi, h, new):
    """The unit's rows, positions and moments before the call, with the
    appended token (position 10**6) when there is one."""
    L = st["lens"][bi, h]
    K, V, pos = st["K"][bi, h, :L], st["V"][bi, h, :L], pos0[bi, h, :L]
    if new:
        K = np.vstack([K, st["kn"][bi, h][None]])
        V = np.vstack([V, st["vn"][bi, h][None]])
        pos = np.append(pos, 10 ** 6)
    m = O.Moments(int(st["n"][bi, h]), st["mu_k"][bi, h], st["mu_v"][bi, h], st["C"][bi, h])
    return K, V, pos, m


def check(gpu, st):
    """Every unit against the oracle following the kernel's evictions;
    returns the number of near ties met."""
    assert gpu["code"] == 0
    G, ties = gpu["G"], 0
    b, H = st["lens"].shape
    for bi in range(b):
        for h in range(H):
            K, V, pos, m = unit_state(st, gpu["pos0"], bi, h, gpu["new"])
            f = check_evicted_unit(gpu, bi, h, st["q"][bi, h * G:(h + 1) * G], K, V, pos, m, gpu["budget"],
                                   gpu["tau"])
            ties += f.ties
    return ties


@pytest.mark.parametrize("new", [False, True])
def test_evict_tiny(new):
    rng = np.random.default_rng(21)
    st = setup(rng, 1, 2, 2, 64, [40, 33], 48, [0, 25])
    gpu = run_case(st, 1, 2, 2, 64, 24, new)
    check(gpu, st)
    if new:
        np.testing.assert_array_equal(gpu["seen"], np.full((1, 2), 10 ** 6 + 1))


@pytest.mark.parametrize("G", [1, 4, 8])
def test_evict_llama_periodic(G):
    """Budget 128 with 64 tokens appended since the last eviction: 64 evictions."""
    rng = np.random.default_rng(22 + G)
    H = 8 if G != 8 else 2
    st = setup(rng, 1, H, G, 128, [191] * H, 200, [2000] * (H // 2) + [0] * (H - H // 2))
    gpu = run_case(st, 1, H, G, 128, 128, True)
    check(gpu, st)


def test_nothing_to_evict_only_appends():
    rng = np.random.default_rng(23)
    st = setup(rng, 2, 2, 2, 64, [10, 3, 0, 7], 16, [0, 1, 2, 3])
    gpu = run_case(st, 2, 2, 2, 64, 12, True)
    check(gpu, st)


def test_capacity_overflow_leaves_unit_unchanged():
    rng = np.random.default_rng(24)
    st = setup(rng, 1, 2, 2, 64, [16, 5], 16, [0, 4])
    gpu = run_case(st, 1, 2, 2, 64, 4, True)
    assert gpu["code"] == 3 and gpu["info"] == 0
    assert gpu["len"][0, 0] == 16 and gpu["len"][0, 1] == 4


@pytest.mark.parametrize("tau", [0.0, 1e-6, 0.05, 0.5])
def test_evict_clamp_paths(tau):
    """Moments from a handful of evicted tokens make n C entries O(1), so a large
    tau clamps a visible share of them: few entries exercise the incremental
    correction list, many exercise the direct clamped product."""
    rng = np.random.default_rng(31)
    st = setup(rng, 1, 2, 2, 64, [60, 45], 64, [3, 5])
    gpu = run_case(st, 1, 2, 2, 64, 30, True, tau=tau)
    check(gpu, st)


def test_evict_large_capacity_fallback():
    """A capacity whose row slices do not fit in shared memory runs the
    single-CTA kernel; results are the same."""
    rng = np.random.default_rng(32)
    st = setup(rng, 1, 1, 4, 128, [2300], 2400, [500])
    gpu = run_case(st, 1, 1, 4, 128, 2260, False)
    check(gpu, st)


def test_evict_budget_zero_and_batch():
    rng = np.random.default_rng(33)
    st = setup(rng, 2, 2, 1, 64, [9, 17, 1, 30], 32, [0, 2, 0, 7])
    gpu = run_case(st, 2, 2, 1, 64, 0, False)
    check(gpu, st)


@pytest.mark.parametrize("cap", [1000, 1200])
def test_evict_slice_sizes(cap):
    """Row slices of 125 rows (register-resident kernel, 9 rows per warp) and
    150 rows (shared-memory cluster kernel): 30 evictions each."""
    rng = np.random.default_rng(34 + cap)
    st = setup(rng, 1, 2, 4, 128, [cap - 11, cap - 20], cap, [300, 0])
    gpu = run_case(st, 1, 2, 4, 128, cap - 41, True)
    check(gpu, st)


def test_evict_many_units():
    """24 units at capacity 200: three waves of 8-CTA clusters of the register
    kernel (5 rows per warp)."""
    rng = np.random.default_rng(27)
    st = setup(rng, 3, 8, 2, 128, [190] * 24, 200, [400, 0] * 12)
    gpu = run_case(st, 3, 8, 2, 128, 140, True)
    check(gpu, st)


def test_periodic_rounds_with_eviction_state():
    """Rounds of 64 appended tokens (mkv_decode_step appends, which leave the
    kept y rows alone) and one mkv_evict_append back to the budget, the cache
    keeping y_j = S_tilde k_j across calls: each round against the oracle
    following the kernel's evictions, and the kept y rows against n C k_j."""
    from test_gpu_decode_evict import check_y_rows
    rng = np.random.default_rng(51)
    b, H, G, D, B, cap, every = 1, 8, 4, 128, 128, 192, 64
    st = setup(rng, b, H, G, D, [B] * H, cap, [4000] * 5 + [0] * 3)
    g = mkv.geom(b, H, G, D)
    pos0 = np.broadcast_to(np.arange(cap, dtype=np.int32) * 3, (b, H, cap)).copy()
    cache = mkv.Cache(bf16(st["K"]), bf16(st["V"]), i32(pos0), i32(st["lens"]), i32(np.full((b, H), 10 ** 6)),
                      torch.zeros(b, H, cap, D, device="cuda"), torch.zeros(b, H, dtype=torch.int32, device="cuda"))
    mom = mkv.Moments(i32(st["n"]), f32(st["mu_k"]), f32(st["mu_v"]), f32(st["C"]))
    ws_d = mkv.alloc_workspace(mkv.mkv_decode_workspace_size(g, cap))
    ws_e = mkv.alloc_workspace(mkv.mkv_evict_workspace_size(g, cap))
    out = torch.empty(b, H * G, D, device="cuda")
    state = {}
    for h in range(H):
        state[h] = dict(K=st["K"][0, h, :B], V=st["V"][0, h, :B], pos=pos0[0, h, :B].astype(np.int64),
                        m=O.Moments(int(st["n"][0, h]), st["mu_k"][0, h], st["mu_v"][0, h], st["C"][0, h]))
    seen = 10 ** 6
    for rnd in range(3):
        kn = bf16_round(1.5 * rng.standard_normal((every, b, H, D)))
        vn = bf16_round(rng.standard_normal((every, b, H, D)))
        q = bf16_round(2.0 * rng.standard_normal((b, H * G, D)))
        for i in range(every):
            mkv.mkv_decode_step(g, bf16(q), bf16(kn[i]), bf16(vn[i]), cache, mom, mkv.mkv_decode_params(1, 1, 1e-6),
                                out, None, ws_d)
        mkv.mkv_evict_append(g, bf16(q), None, None, B, cache, mom, 1e-6, ws_e)
        assert mkv.mkv_get_device_error(ws_d)[0] == 0 and mkv.mkv_get_device_error(ws_e)[0] == 0
        gpu = dict(K=host(cache.K), V=host(cache.V), pos=host(cache.pos), len=host(cache.len), n=host(mom.n),
                   mu_k=host(mom.mu_k), mu_v=host(mom.mu_v), C=host(mom.C))
        assert (host(cache.y_len) == B).all()
        for h in range(H):
            s0 = state[h]
            K = np.vstack([s0["K"], kn[:, 0, h]])
            V = np.vstack([s0["V"], vn[:, 0, h]])
            pos = np.append(s0["pos"], seen + np.arange(every))
            f = check_evicted_unit(gpu, 0, h, q[0, h * G:(h + 1) * G], K, V, pos, s0["m"], B, 1e-6)
            state[h] = dict(K=f.K, V=f.V, pos=f.pos, m=f.moments)
        seen += every
        check_y_rows(cache, mom)


def test_eviction_state_reset_by_compress_and_large_capacity():
    """mkv_compress leaves no y row current; the eviction kernel for
    capacities past the register kernel's does not keep y either."""
    from paper_2606_01563_gb300.inputs import WORKLOADS, Generator
    wl = WORKLOADS["tiny_d64_t1k"]
    K, V, Q = Generator(wl, seed=2).prefill()
    G_ = wl.geom
    g = mkv.geom(G_.batch, G_.n_kv_heads, G_.group, G_.head_dim)
    cache = mkv.alloc_cache(g, wl.budget + 4, evict_state=True)
    cache.y_len.fill_(7)
    p = mkv.mkv_compress_params(wl.budget, wl.window, 1, 1, 1, 1, 1, 1e-6)
    ws = mkv.alloc_workspace(mkv.mkv_compress_workspace_size(g, wl.T, p))
    mkv.mkv_compress(g, wl.T, bf16(K), bf16(V), bf16(Q), p, cache, mkv.alloc_moments(g), ws)
    assert mkv.mkv_get_device_error(ws)[0] == 0
    assert (host(cache.y_len) == 0).all()
    # capacity 2400 runs the single-CTA kernel: y_len goes to 0 after its evictions
    rng = np.random.default_rng(32)
    st = setup(rng, 1, 1, 4, 128, [2300], 2400, [500])
    g = mkv.geom(1, 1, 4, 128)
    pos0 = np.arange(2400, dtype=np.int32)[None, None] * 3
    c = mkv.Cache(bf16(st["K"]), bf16(st["V"]), i32(pos0), i32(st["lens"]), i32(np.full((1, 1), 10 ** 6)),
                  torch.zeros(1, 1, 2400, 128, device="cuda"), torch.full((1, 1), 2300, dtype=torch.int32, device="cuda"))
    mom = mkv.Moments(i32(st["n"]), f32(st["mu_k"]), f32(st["mu_v"]), f32(st["C"]))
    ws = mkv.alloc_workspace(mkv.mkv_evict_workspace_size(g, 2400))
    mkv.mkv_evict_append(g, bf16(st["q"]), None, None, 2290, c, mom, 1e-6, ws)
    assert mkv.mkv_get_device_error(ws)[0] == 0
    assert int(host(c.y_len)[0, 0]) == 0 and int(host(c.len)[0, 0]) == 2290
