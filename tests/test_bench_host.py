"""Host logic of bench.py that needs no GPU: the code hash that decides
whether the committed ncu DRAM traffic still describes the timed kernel."""
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402

SRC = r'''// header comment
#include "common.cuh"
/* block
   comment */
__global__ void k(float* x) {
  const char* s = "a // not a comment";  // trailing
  char c = '"';
  x[threadIdx.x] = 1.0f;
}
'''


def _sha(tmp_path, text, name="k.cu"):
    p = tmp_path / name
    p.write_text(text)
    return bench.code_sha([str(p)])


def test_code_sha_ignores_comments_and_spacing(tmp_path):
    base = _sha(tmp_path, SRC)
    edited = SRC.replace("// header comment", "// another header\n// over two lines")
    edited = edited.replace("/* block\n   comment */", "/* shorter */")
    edited = edited.replace("x[threadIdx.x] = 1.0f;", "x[threadIdx.x]   =   1.0f;")
    assert _sha(tmp_path, edited) == base


def test_code_sha_sees_code_and_literals(tmp_path):
    base = _sha(tmp_path, SRC)
    assert _sha(tmp_path, SRC.replace("threadIdx.x", "threadIdx.y")) != base
    # text after // inside a string literal is code, not a comment
    assert _sha(tmp_path, SRC.replace("not a comment", "not a remark")) != base
    assert _sha(tmp_path, SRC.replace("'\"'", "'x'")) != base


def test_kernel_sources_exist():
    for cu in ("decode_cl.cu", "decode.cu", "compress.cu", "evict.cu"):
        paths = bench.kernel_sources(cu)
        assert all(os.path.exists(p) for p in paths)
        assert len(bench.code_sha(paths)) == 64


def _fake_run(name, B, S, L=1, evict_every=0):
    """A bench.Run holding only what the byte accounting reads (no GPU state)."""
    from paper_2606_01563_gb300.inputs import WORKLOADS
    st = type("FakeStack", (), {})()
    st.wl = WORKLOADS[name]
    st.G, st.S, st.L = st.wl.geom, S, L
    r = bench.Run.__new__(bench.Run)
    r.st, r.G, r.B, r.ev_every = st, st.G, B, evict_every
    return r


def test_decode_bytes_per_launch():
    # Llama-3.1-8B geometry, batch 1: 8 units, 32 query heads, d = 128
    units, hq, d = 8, 32, 128
    retained = units * 256 * d * 2 * 2          # K and V rows, bf16
    moments = units * (d * d * 4 + 2 * d * 4 + 4)  # C, mu_k, mu_v, n
    q, out = hq * d * 2, hq * d * 4
    assert retained + moments + q + out == 1605664  # 1.61 MB at budget 256
    new_row = units * d * 2 * 2                  # k_new, v_new read, and the row written
    assert _fake_run("llama8b_layer_t8k", 256, 1).decode_bytes() == 1605664 + 2 * new_row
    # 256 launches over 512..575 rows (an eviction back to 512 every 64)
    assert _fake_run("llama8b_layer_t8k", 512, 256, evict_every=64).decode_bytes() / 256 == 2791456
    # the headline at budget 1024: 36 layers, 512 steps over 1024..1535 rows, batch 4 (32 units, 128 q heads)
    r = _fake_run("qwen4b_t32k", 1024, 512, L=36)
    units, hq = 32, 128
    per_row = units * d * 4
    fixed = units * (d * d * 4 + 2 * d * 4 + 4) + hq * d * (2 + 4) + 2 * units * d * 4
    want = 36 * sum(fixed + (1024 + i) * per_row for i in range(512))
    assert r.decode_bytes() == want
    assert abs(want / (36 * 512) - 23.22e6) < 0.01e6


def test_compress_bytes():
    units, d, T, B, g, w = 8, 128, 8192, 512, 4, 32
    want = units * (2 * T * d * 2 + g * w * d * 2 + B * (d * 2 * 2 + 4) + (d * d + 2 * d + 1) * 4)
    assert _fake_run("llama8b_layer_t8k", B, 256).compress_bytes() == want == 36462624
    # the headline layer at 32K, batch 4: 537 MB of K and V dominate
    assert abs(_fake_run("qwen4b_t32k", 1024, 512).compress_bytes() - 557.0e6) < 0.1e6


def test_oracle_sample_stands_for_its_share_of_the_step():
    from paper_2606_01563_gb300.inputs import WORKLOADS
    wl = WORKLOADS["qwen4b_t32k"]
    # 16 of the step's 36 x 32 (layer, unit) jobs per budget; each budget makes 4 x 512 tokens
    assert bench.step_tokens_equiv(wl, 36, 16) == 16 * 4 * 512 / (36 * 32)
    cfg = bench.config_dict(36)
    assert cfg["layers"] == 36 and cfg["budgets"] == [128, 256, 1024] and cfg["seq_len"] == 32768
    assert cfg["decode_steps"] == 512 and cfg["global_batch"] == 4


def test_oracle_jobs_rotate_units_and_budgets():
    import torch
    from paper_2606_01563_gb300.inputs import WORKLOADS, TorchGenerator
    wl = WORKLOADS["tiny_d64_t1k"]
    gen = TorchGenerator(wl, seed=0)
    K, V, Q = gen.prefill()
    q, kn, vn = gen.decode(3)
    st = type("S", (), {})()
    st.G, st.wl, st.L = wl.geom, wl, 1
    st.K, st.V, st.Q, st.q, st.kn, st.vn = [K], [V], [Q], q[:, None], kn[:, None], vn[:, None]
    jobs = bench.oracle_jobs_from_stack(st, 4)
    assert [j[6] for j in jobs] == [128, 256, 1024, 128]
    # unit 1 = (batch 0, KV head 1): its rows and its group's query heads 2..3
    assert torch.equal(torch.from_numpy(jobs[1][0]), K[0, 1].float())
    assert torch.equal(torch.from_numpy(jobs[1][3]), q[:, 0, 2:4].float())
    assert jobs[0][3].shape == (3, 2, 64) and jobs[0][4].shape == (3, 64)
    nxt = bench.oracle_jobs_from_stack(st, 4, step=1)
    assert [j[6] for j in nxt] == [256, 1024, 128, 256]


class _FakeProc:
    def __init__(self, out):
        self.out = out

    def terminate(self):
        pass

    def communicate(self, timeout=None):
        return self.out, ""

    def kill(self):
        pass


def test_clock_samples_and_throttle_reasons():
    c = bench.Clocks(0)
    c.proc = _FakeProc("2070, 2070, 900.1, Not Active, Not Active, Not Active, Not Active\n"
                       "2055, 2070, 1390.0, Not Active, Not Active, Not Active, Active\n"
                       "2070, 2070, 1000.0, Not Active, Not Active, Not Active, Not Active\n"
                       "[N/A], 2070, 1000.0, Not Active, Not Active, Not Active, Not Active\n")
    r = c.stop()
    assert r["sm_mhz"] == 2070.0 and r["sm_max_mhz"] == 2070.0 and r["samples"] == 3
    assert r["reasons"] == ["sw_power_cap"]
    c.proc = _FakeProc("1500, 2070, 800.0, Active, Not Active, Active, Not Active\n")
    assert bench.Clocks.stop(c)["reasons"] == ["hw_slowdown", "sw_thermal_slowdown"]
    c.proc = None
    assert c.stop()["sm_mhz"] is None


class _CountingBinding:
    """Stands in for the binding: counts the kernels each entry point launches
    (a per-unit compress with T > budget: 9; a decode step, an eviction and a
    pack of C': 1 each)."""
    KERNELS = {"mkv_compress": 9, "mkv_decode_step": 1, "mkv_evict_append": 1, "mkv_moments_pack_split": 1}

    def __init__(self):
        self.launched = 0
        self.calls = []

    def __getattr__(self, name):
        def call(*args, **kwargs):
            self.calls.append(name)
            self.launched += self.KERNELS[name]
        return call


class _Index:
    def __getitem__(self, key):
        return None


def test_launch_count_matches_the_parts():
    """Run.launches() (the bench's gpu_launches claim) equals the kernels one
    pass over the run's parts launches, with and without periodic eviction."""
    from paper_2606_01563_gb300.inputs import WORKLOADS
    for name, B, S, L, every in (("qwen4b_t32k", 128, 512, 3, 0), ("llama8b_t128k", 128, 1024, 2, 64),
                                 ("llama8b_layer_t8k", 512, 256, 1, 64)):
        st = type("FakeStack", (), {})()
        st.wl = WORKLOADS[name]
        st.G, st.S, st.L = st.wl.geom, S, L
        st.K = st.V = st.Q = [None] * L
        st.q = st.kn = st.vn = _Index()
        r = bench.Run.__new__(bench.Run)
        fake = _CountingBinding()
        r.mkv, r.st, r.G, r.B, r.ev_every = fake, st, st.G, B, every
        r.block = every if every else 64
        r.g = r.p = r.ws_c = r.ws_d = r.ws_e = r.out = None
        r.caches, r.moms, r.csplit, r.dps = [None] * L, [None] * L, [None] * L, [None] * L
        r.final = [None] * S
        for _, fn in r.parts(st):
            fn()
        assert fake.launched == r.launches(), (name, fake.launched, r.launches())
        # every change of the moments is followed by a pack of that layer's C'
        changes = sum(c in ("mkv_compress", "mkv_evict_append") for c in fake.calls)
        assert fake.calls.count("mkv_moments_pack_split") == changes


def test_twin_input_set_is_a_distinct_copy():
    """The end-to-end leg's second input set: the same shapes and contents as
    the first in separate storage (CPU tensors stand in for device ones)."""
    import torch
    from paper_2606_01563_gb300.inputs import WORKLOADS
    st = bench.Stack.__new__(bench.Stack)
    st.wl = WORKLOADS["llama8b_layer_t8k"]
    st.G, st.L, st.S = st.wl.geom, 2, 4
    g = torch.Generator().manual_seed(0)
    rnd = lambda *s: torch.randn(*s, generator=g).bfloat16()
    st.K, st.V, st.Q = [rnd(1, 2, 16, 8) for _ in range(2)], [rnd(1, 2, 16, 8) for _ in range(2)], \
        [rnd(1, 2, 4, 8) for _ in range(2)]
    st.q, st.kn, st.vn = rnd(4, 2, 1, 8, 8), rnd(4, 2, 1, 2, 8), rnd(4, 2, 1, 2, 8)
    tw = st.twin()
    assert (tw.wl, tw.G, tw.L, tw.S) == (st.wl, st.G, st.L, st.S)
    assert tw.nbytes() == st.nbytes()
    for a, b in zip(st.tensors(), tw.tensors()):
        assert torch.equal(a, b) and a.data_ptr() != b.data_ptr()
