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
