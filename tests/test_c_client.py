"""The boundary is a plain C ABI: a C99 program that includes include/mkv.h
and links libmkv.so compiles, sees the struct layouts the Python binding
assumes, and gets the documented status codes from host-side validation.
Nothing is launched (every call is rejected before any kernel), so this
runs on the CPU.  The header must also compile as C++."""
import os
import shutil
import subprocess

import pytest

from paper_2606_01563_gb300 import mkv

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
INCLUDE = os.path.join(ROOT, "include")
LIBDIR = os.path.dirname(mkv.LIB_PATH)

CLIENT = r"""
#include <stddef.h>
#include <stdint.h>
#include <stdio.h>
#include <string.h>

#include "mkv.h"

/* never dereferenced: every call below is rejected before it touches memory */
#define FAKE ((void*)(uintptr_t)(1u << 20))

static int fails = 0;
#define CHECK(cond)                                        \
  do {                                                     \
    if (!(cond)) {                                         \
      printf("FAIL line %d: %s\n", __LINE__, #cond);       \
      ++fails;                                             \
    }                                                      \
  } while (0)

int main(void) {
  const mkv_geom g = {1, 2, 4, 128};
  const mkv_geom bad_dim = {1, 2, 4, 96};
  const mkv_geom bad_group = {1, 2, 3, 128};
  mkv_cache c = {FAKE, FAKE, (int32_t*)FAKE, (int32_t*)FAKE, (int32_t*)FAKE, 64, NULL, NULL};
  mkv_moments m = {(int32_t*)FAKE, (float*)FAKE, (float*)FAKE, (float*)FAKE};
  mkv_decode_params dp = {1, 1, 1e-6f, NULL, 0, NULL};
  mkv_compress_params cp = {128, 16, 1, 1, 1, 1, 1, 1e-6f, 0};
  mkv_compress_params small = cp;
  const size_t big = (size_t)1 << 30;

  /* layouts (LP64) as the Python binding declares them */
  CHECK(sizeof(mkv_geom) == 16);
  CHECK(sizeof(mkv_moments) == 32);
  CHECK(sizeof(mkv_cache) == 64 && offsetof(mkv_cache, capacity) == 40 && offsetof(mkv_cache, y_len) == 56);
  CHECK(sizeof(mkv_compress_params) == 36);
  CHECK(offsetof(mkv_compress_params, tau) == 28 && offsetof(mkv_compress_params, adaptive) == 32);
  CHECK(sizeof(mkv_decode_params) == 40 && offsetof(mkv_decode_params, C16) == 16 &&
        offsetof(mkv_decode_params, early_load) == 24 && offsetof(mkv_decode_params, C_split) == 32);
  CHECK(sizeof(mkv_compress_diag) == 24);
  CHECK(sizeof(mkv_status) == 4 && MKV_ERR_WORKSPACE == 7);

  CHECK(mkv_version() == 202);
  CHECK(strcmp(mkv_status_str(MKV_OK), "ok") == 0);
  CHECK(strcmp(mkv_status_str((mkv_status)99), "unknown status") == 0);

  /* decode */
  CHECK(mkv_decode_step(bad_dim, FAKE, NULL, NULL, &c, &m, &dp, (float*)FAKE, NULL, FAKE, big, NULL) ==
        MKV_ERR_UNSUPPORTED);
  CHECK(mkv_decode_step(bad_group, FAKE, NULL, NULL, &c, &m, &dp, (float*)FAKE, NULL, FAKE, big, NULL) ==
        MKV_ERR_SHAPE);
  CHECK(mkv_decode_step(g, NULL, NULL, NULL, &c, &m, &dp, (float*)FAKE, NULL, FAKE, big, NULL) ==
        MKV_ERR_INVALID_ARG);
  CHECK(mkv_decode_step(g, FAKE, FAKE, NULL, &c, &m, &dp, (float*)FAKE, NULL, FAKE, big, NULL) ==
        MKV_ERR_INVALID_ARG);
  CHECK(mkv_decode_step(g, FAKE, NULL, NULL, &c, &m, &dp, (float*)FAKE, NULL, NULL, big, NULL) ==
        MKV_ERR_WORKSPACE);
  CHECK(mkv_decode_step_noalloc(bad_dim, FAKE, NULL, NULL, &c, &m, &dp, (float*)FAKE, NULL, NULL) ==
        MKV_ERR_UNSUPPORTED);
  CHECK(mkv_moments_pack_bf16(g, &m, NULL, NULL) == MKV_ERR_INVALID_ARG);
  CHECK(mkv_moments_pack_split(g, &m, 1e-6f, NULL, NULL) == MKV_ERR_INVALID_ARG);

  /* compress */
  CHECK(mkv_compress_workspace_size(g, 1024, &cp) > 0);
  small.budget = 10; /* below sink + window */
  CHECK(mkv_compress_workspace_size(g, 1024, &small) == 0);
  CHECK(mkv_compress(g, 1024, FAKE, FAKE, FAKE, &small, &c, &m, NULL, FAKE, big, NULL) == MKV_ERR_INVALID_ARG);
  c.capacity = 100; /* below the budget */
  CHECK(mkv_compress(g, 1024, FAKE, FAKE, FAKE, &cp, &c, &m, NULL, FAKE, big, NULL) == MKV_ERR_CAPACITY);
  c.capacity = 64;

  /* eviction */
  CHECK(mkv_evict_append(g, FAKE, NULL, NULL, -1, &c, &m, 0.f, FAKE, big, NULL) == MKV_ERR_INVALID_ARG);
  CHECK(mkv_evict_workspace_size(g, 70000) == 0);
  CHECK(mkv_decode_evict_step(g, FAKE, NULL, NULL, 8, &c, &m, &dp, (float*)FAKE, NULL, FAKE, big, NULL) ==
        MKV_ERR_INVALID_ARG);
  CHECK(mkv_get_device_error(NULL, NULL, NULL) == MKV_ERR_WORKSPACE);

  printf("%s\n", fails ? "FAILED" : "ok");
  return fails != 0;
}
"""


@pytest.fixture(scope="module")
def lib_built():
    if not os.path.exists(mkv.LIB_PATH):
        from paper_2606_01563_gb300 import build
        build.build()
    return mkv.LIB_PATH


def _cc():
    for c in ("gcc", "cc"):
        if shutil.which(c):
            return c
    pytest.skip("no C compiler")


def test_c99_client_links_and_validates(lib_built, tmp_path):
    src = tmp_path / "client.c"
    src.write_text(CLIENT)
    exe = tmp_path / "client"
    r = subprocess.run([_cc(), "-std=c99", "-Wall", "-Wextra", "-Werror", "-pedantic", "-I", INCLUDE, str(src),
                        "-o", str(exe), "-L", LIBDIR, "-lmkv", f"-Wl,-rpath,{LIBDIR}"],
                       capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0 and r.stdout.strip().endswith("ok"), r.stdout + r.stderr


def test_header_compiles_as_cpp(tmp_path):
    cxx = shutil.which("g++") or shutil.which("c++")
    if cxx is None:
        pytest.skip("no C++ compiler")
    src = tmp_path / "h.cpp"
    src.write_text('#include "mkv.h"\nint main() { return mkv_version() == 202 ? 0 : 1; }\n')
    r = subprocess.run([cxx, "-std=c++17", "-Wall", "-Wextra", "-Werror", "-fsyntax-only", "-I", INCLUDE, str(src)],
                       capture_output=True, text=True)
    assert r.returncode == 0, r.stderr


def test_binding_structs_match_the_c_layout():
    import ctypes
    assert ctypes.sizeof(mkv.mkv_geom) == 16
    assert ctypes.sizeof(mkv.mkv_moments) == 32
    assert ctypes.sizeof(mkv.mkv_cache) == 64 and mkv.mkv_cache.capacity.offset == 40
    assert mkv.mkv_cache.y.offset == 48 and mkv.mkv_cache.y_len.offset == 56
    assert ctypes.sizeof(mkv.mkv_compress_params) == 36
    assert mkv.mkv_compress_params.tau.offset == 28 and mkv.mkv_compress_params.adaptive.offset == 32
    assert ctypes.sizeof(mkv.mkv_decode_params) == 40 and mkv.mkv_decode_params.C16.offset == 16
    assert mkv.mkv_decode_params.early_load.offset == 24 and mkv.mkv_decode_params.C_split.offset == 32
    assert ctypes.sizeof(mkv.mkv_compress_diag) == 24
