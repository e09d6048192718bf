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
    for cu in ("decode.cu", "compress.cu", "evict.cu"):
        paths = bench.kernel_sources(cu)
        assert all(os.path.exists(p) for p in paths)
        assert len(bench.code_sha(paths)) == 64


def _fake_step(B, S, T=8192):
    """A bench.Step holding only what the byte accounting reads (no GPU state)."""
    from paper_2606_01563_gb300.inputs import WORKLOADS
    st = bench.Step.__new__(bench.Step)
    st.wl = WORKLOADS[bench.WORKLOAD]
    st.G = st.wl.geom
    st.B, st.S, st.T = B, S, T
    return st


def test_decode_bytes_per_launch():
    # Llama-3.1-8B geometry, batch 1: 8 units, 32 query heads, d = 128
    units, hq, d = 8, 32, 128
    retained = units * 256 * d * 2 * 2          # K and V rows, bf16
    moments = units * (d * d * 4 + 2 * d * 4 + 4)  # C, mu_k, mu_v, n
    q, out = hq * d * 2, hq * d * 4
    assert retained + moments + q + out == 1605664  # 1.61 MB at budget 256
    new_row = units * d * 2 * 2                  # k_new, v_new read, and the row written
    assert _fake_step(256, 1).decode_bytes_total() == 1605664 + 2 * new_row
    # the bench step: 256 launches over 512..575 rows (an eviction back to 512 every 64)
    assert _fake_step(512, 256).decode_bytes_total() / 256 == 2791456


def test_compress_bytes():
    units, d, T, B, g, w = 8, 128, 8192, 512, 4, 32
    want = units * (2 * T * d * 2 + g * w * d * 2 + B * d * 2 * 2 + (d * d + 2 * d + 1) * 4)
    assert _fake_step(B, 256, T).compress_bytes() == want == 36446240


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
