"""The C-ABI library builds, loads and exports every entry point include/mkv.h
declares; host-side validation rejects bad arguments before touching the
GPU.  Runs on the CPU (no kernel is launched)."""
import ctypes
import os
import re

import pytest

from paper_2606_01563_gb300 import mkv

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    if not os.path.exists(mkv.LIB_PATH):
        from paper_2606_01563_gb300 import build
        build.build()
    return mkv.lib()


def declared_functions(header="mkv.h"):
    src = open(os.path.join(ROOT, "include", header)).read()
    return sorted(set(re.findall(r"MKV_API\s+[\w\s\*]+?\b(mkv_\w+)\s*\(", src)))


def test_every_declared_symbol_is_exported(L):
    names = declared_functions()
    assert len(names) == 14, names
    assert set(names) == set(mkv.EXPORTS)
    for n in names:
        assert hasattr(L, n), n
    debug = declared_functions("mkv_debug.h")
    assert set(debug) == set(mkv.DEBUG_EXPORTS) and len(debug) == 2
    for n in debug:
        assert hasattr(L, n), n


def test_debug_hooks_round_trip(L):
    """The test hooks only set process-wide values read at the next launch."""
    default = mkv.mkv_debug_set_poll_limit(5)
    assert default == 1 << 22
    assert mkv.mkv_debug_set_poll_limit(-1) == 5
    assert mkv.mkv_debug_set_poll_limit(-1) == default
    assert mkv.mkv_debug_force_ticket_merge(1) == 0
    assert mkv.mkv_debug_force_ticket_merge(0) == 1


def test_version_and_status_strings(L):
    assert mkv.mkv_version() == 202
    for code in range(8):
        assert mkv.mkv_status_str(code)
    assert mkv.mkv_status_str(99) == "unknown status"


FAKE = 1 << 20  # never dereferenced: validation fails before any launch


def fake_cache(cap=64):
    return mkv.mkv_cache(FAKE, FAKE, FAKE, FAKE, FAKE, cap)


def fake_moments():
    return mkv.mkv_moments(FAKE, FAKE, FAKE, FAKE)


def decode(L, g, q=FAKE, kn=None, vn=None, cache=None, mom=None, p=None, out=FAKE, ws=FAKE, wsb=1 << 30):
    cache = cache or fake_cache()
    mom = mom or fake_moments()
    p = p or mkv.mkv_decode_params(1, 1, 1e-6)
    return L.mkv_decode_step(g, q, kn, vn, ctypes.byref(cache), ctypes.byref(mom), ctypes.byref(p), out, None,
                             ws, wsb, None)


def test_decode_validation(L):
    g = mkv.geom(1, 2, 4, 128)
    assert decode(L, mkv.geom(1, 2, 4, 96)) == 6            # head_dim unsupported
    assert decode(L, mkv.geom(1, 2, 3, 128)) == 2           # group unsupported
    assert decode(L, mkv.geom(0, 2, 4, 128)) == 2           # empty batch
    assert decode(L, mkv.geom(65536, 1, 4, 128)) == 2       # batch past the grid's z limit
    assert decode(L, mkv.geom(1, 65536, 4, 128)) == 2       # KV heads past the grid's y limit
    assert decode(L, g, q=None) == 1
    assert decode(L, g, out=None) == 1
    assert decode(L, g, kn=FAKE) == 1                        # k_new without v_new
    assert decode(L, g, p=mkv.mkv_decode_params(1, 2, 0.0)) == 1   # order
    assert decode(L, g, p=mkv.mkv_decode_params(1, 1, -1.0)) == 1  # tau
    assert decode(L, g, cache=mkv.mkv_cache(FAKE, FAKE, FAKE, FAKE, FAKE, 0)) == 1
    assert decode(L, g, cache=mkv.mkv_cache(FAKE + 2, FAKE, FAKE, FAKE, FAKE, 64)) == 1  # misaligned K
    assert decode(L, g, cache=mkv.mkv_cache(FAKE, FAKE, FAKE, FAKE, FAKE, 64, FAKE, None)) == 1  # y without y_len
    assert decode(L, g, cache=mkv.mkv_cache(FAKE, FAKE, FAKE, FAKE, FAKE, 64, None, FAKE)) == 1  # y_len without y
    assert decode(L, g, cache=mkv.mkv_cache(FAKE, FAKE, FAKE, FAKE, FAKE, 64, FAKE + 8, FAKE)) == 1  # misaligned y
    assert decode(L, g, ws=None) == 7
    assert decode(L, g, wsb=16) == 7
    assert decode(L, g, ws=FAKE + 8) == 7                    # misaligned workspace
    assert decode(L, g, p=mkv.mkv_decode_params(1, 1, 0.0, FAKE + 8)) == 1  # misaligned bf16 C copy
    assert decode(L, g, p=mkv.mkv_decode_params(1, 1, 0.0, None, 0, FAKE + 8)) == 1  # misaligned operand form
    assert decode(L, g, p=mkv.mkv_decode_params(1, 1, 0.0, FAKE, 0, FAKE)) == 1  # operand form with the bf16 copy
    assert decode(L, g, q=FAKE + 4) == 1                     # misaligned q
    assert decode(L, g, p=mkv.mkv_decode_params(1, 1, 0.0, None, 2)) == 1   # early_load not 0/1
    # mu_k is read as float2 and mu_v as float4: 4-byte alignment is not enough
    assert decode(L, g, mom=mkv.mkv_moments(FAKE, FAKE + 4, FAKE, FAKE)) == 1
    assert decode(L, g, mom=mkv.mkv_moments(FAKE, FAKE, FAKE + 8, FAKE)) == 1
    assert decode(L, g, mom=mkv.mkv_moments(FAKE, FAKE, FAKE, FAKE + 8)) == 1
    # without the correction the moments are not read, so they are not checked
    assert decode(L, g, mom=mkv.mkv_moments(FAKE, FAKE + 4, FAKE, FAKE), p=mkv.mkv_decode_params(0, 1, 0.0),
                  wsb=16) == 7


def noalloc(L, g, q=FAKE, cache=None, mom=None, p=None, out=FAKE):
    cache = cache or fake_cache()
    mom = mom or fake_moments()
    p = p or mkv.mkv_decode_params(1, 1, 1e-6)
    return L.mkv_decode_step_noalloc(g, q, None, None, ctypes.byref(cache), ctypes.byref(mom), ctypes.byref(p),
                                     out, None, None)


def test_noalloc_validation_matches_decode(L):
    """The no-allocation decode rejects what mkv_decode_step rejects, with the
    same status, before it touches the device (these cases never get there)."""
    g = mkv.geom(1, 2, 4, 128)
    cases = [dict(g=mkv.geom(1, 2, 4, 96)), dict(g=mkv.geom(1, 2, 3, 128)), dict(g=mkv.geom(65536, 1, 4, 128)),
             dict(g=mkv.geom(1, 65536, 4, 128)), dict(q=None), dict(out=FAKE + 8),
             dict(mom=mkv.mkv_moments(FAKE, FAKE + 4, FAKE, FAKE)),
             dict(mom=mkv.mkv_moments(FAKE, FAKE, FAKE + 8, FAKE)),
             dict(cache=mkv.mkv_cache(FAKE + 2, FAKE, FAKE, FAKE, FAKE, 64)),
             dict(p=mkv.mkv_decode_params(1, 2, 0.0)), dict(p=mkv.mkv_decode_params(1, 1, 0.0, FAKE + 8)),
             dict(p=mkv.mkv_decode_params(1, 1, 0.0, None, 0, FAKE + 4))]
    for kw in cases:
        gg = kw.pop("g", g)
        want = decode(L, gg, **kw)
        assert want in (1, 2, 6), kw
        assert noalloc(L, gg, **kw) == want, kw
    # more units than the fixed scratch holds even at one split per unit
    assert noalloc(L, mkv.geom(64, 256, 8, 128)) == 7


def test_pack_bf16_validation(L):
    g = mkv.geom(1, 2, 4, 128)
    m = mkv.mkv_moments(FAKE, FAKE, FAKE, FAKE)
    assert L.mkv_moments_pack_bf16(g, ctypes.byref(m), None, None) == 1
    assert L.mkv_moments_pack_bf16(g, ctypes.byref(m), FAKE + 8, None) == 1
    assert L.mkv_moments_pack_bf16(g, None, FAKE, None) == 1
    assert L.mkv_moments_pack_bf16(mkv.geom(1, 2, 4, 96), ctypes.byref(m), FAKE, None) == 6


def test_pack_split_validation(L):
    g = mkv.geom(1, 2, 4, 128)
    m = mkv.mkv_moments(FAKE, FAKE, FAKE, FAKE)
    assert L.mkv_moments_pack_split(g, ctypes.byref(m), 1e-6, None, None) == 1
    assert L.mkv_moments_pack_split(g, ctypes.byref(m), 1e-6, FAKE + 8, None) == 1
    assert L.mkv_moments_pack_split(g, ctypes.byref(m), -1.0, FAKE, None) == 1
    assert L.mkv_moments_pack_split(g, ctypes.byref(m), float("nan"), FAKE, None) == 1
    assert L.mkv_moments_pack_split(g, None, 1e-6, FAKE, None) == 1
    assert L.mkv_moments_pack_split(g, ctypes.byref(mkv.mkv_moments(FAKE, FAKE, FAKE, FAKE + 8)), 1e-6, FAKE,
                                    None) == 1  # C misaligned
    assert L.mkv_moments_pack_split(mkv.geom(1, 2, 4, 96), ctypes.byref(m), 1e-6, FAKE, None) == 6


def test_workspace_sizes(L):
    g = mkv.geom(2, 8, 4, 128)
    assert L.mkv_decode_workspace_size(g, 576) > 256
    assert L.mkv_decode_workspace_size(mkv.geom(2, 8, 4, 80), 576) == 0
    assert L.mkv_evict_workspace_size(g, 576) >= 256 + 2 * 8 * 4 * 576 * 4
    assert L.mkv_evict_workspace_size(g, 70000) == 0
    p = mkv.mkv_compress_params(512, 32, 1, 1, 1, 1, 1, 1e-6)
    assert L.mkv_compress_workspace_size(g, 8192, ctypes.byref(p)) > 2 * 8 * 8192 * 4
    bad = mkv.mkv_compress_params(16, 32, 1, 1, 1, 1, 1, 1e-6)  # budget < protected
    assert L.mkv_compress_workspace_size(g, 8192, ctypes.byref(bad)) == 0


def compress(L, g, T, p, cache=None, ws=FAKE, wsb=1 << 30, K=FAKE):
    cache = cache or fake_cache(1024)
    mom = fake_moments()
    return L.mkv_compress(g, T, K, FAKE, FAKE, ctypes.byref(p), ctypes.byref(cache), ctypes.byref(mom), None,
                          ws, wsb, None)


def test_compress_validation(L):
    g = mkv.geom(1, 2, 2, 64)
    P = lambda **kw: mkv.mkv_compress_params(**{**dict(budget=128, window=16, sink=1, keep_window=1, pool=1,
                                                        mi=1, causal=1, tau=1e-6), **kw})
    assert compress(L, g, 1024, P(budget=10)) == 1            # budget below sink + window
    assert compress(L, g, 1024, P(window=0)) == 1
    assert compress(L, g, 8, P(window=16)) == 1               # window longer than the prompt
    assert compress(L, mkv.geom(1, 2, 4, 64), 1024, P(budget=200, window=65)) == 2  # 260 window rows
    assert compress(L, mkv.geom(256, 256, 2, 64), 1024, P()) == 2   # 65536 units: one grid row each
    assert compress(L, g, 1024, P(pool=3)) == 1
    assert compress(L, g, 1024, P(mi=2)) == 1
    assert compress(L, g, 0, P()) == 1
    assert compress(L, g, 1024, P(), cache=fake_cache(100)) == 3   # capacity < budget
    assert compress(L, g, 1024, P(), K=None) == 1
    assert compress(L, g, 1024, P(), wsb=1024) == 7
    assert compress(L, mkv.geom(1, 2, 2, 100), 1024, P()) == 6
    # adaptive budget: a head may keep 17 protected rows plus all 2 * 111 joint selections
    assert compress(L, g, 1024, P(adaptive=2)) == 1
    assert compress(L, g, 1024, P(adaptive=1), cache=fake_cache(238)) == 3
    assert compress(L, g, 1024, P(adaptive=1), cache=fake_cache(239), wsb=1024) == 7
    assert compress(L, g, 200, P(adaptive=1), cache=fake_cache(199), wsb=1024) == 3   # min(T, ...) = T
    assert compress(L, mkv.geom(1, 65, 2, 64), 1024, P(adaptive=1)) == 2
    ws0 = L.mkv_compress_workspace_size(g, 1024, ctypes.byref(P()))
    ws1 = L.mkv_compress_workspace_size(g, 1024, ctypes.byref(P(adaptive=1)))
    assert ws1 > ws0 > 0


def test_decode_evict_validation(L):
    g = mkv.geom(1, 2, 2, 64)
    c, m = fake_cache(), fake_moments()
    P = lambda **kw: mkv.mkv_decode_params(**{**dict(correction=1, order=1, tau=1e-6, C16=None), **kw})

    def run(**kw):
        p = kw.get("p", P())
        return L.mkv_decode_evict_step(kw.get("g", g), kw.get("q", FAKE), kw.get("kn", FAKE), FAKE,
                                       kw.get("budget", 8), ctypes.byref(c), ctypes.byref(m), ctypes.byref(p),
                                       kw.get("out", FAKE), None, kw.get("ws", FAKE), kw.get("wsb", 1 << 30), None)
    assert run(budget=-1) == 1
    assert run(q=None) == 1
    assert run(kn=None) == 1                      # the token to append is required
    assert run(out=FAKE + 8) == 1                 # misaligned output
    assert run(p=P(order=2)) == 1
    assert run(p=P(C16=FAKE)) == 1                # a 16-bit copy of C would be stale
    assert run(p=P(C_split=FAKE)) == 1            # so would the operand form of C'
    assert run(wsb=8) == 7
    assert run(g=mkv.geom(1, 2, 5, 64)) == 2
    n = L.mkv_decode_evict_workspace_size(g, 64)
    assert n >= L.mkv_evict_workspace_size(g, 64) and n >= L.mkv_decode_workspace_size(g, 64)
    assert L.mkv_decode_evict_workspace_size(g, 0) == 0


def test_evict_validation(L):
    g = mkv.geom(1, 2, 2, 64)
    c, m = fake_cache(), fake_moments()
    run = lambda **kw: L.mkv_evict_append(kw.get("g", g), kw.get("q", FAKE), None, None, kw.get("budget", 8),
                                          ctypes.byref(c), ctypes.byref(m), kw.get("tau", 0.0),
                                          kw.get("ws", FAKE), kw.get("wsb", 1 << 30), None)
    assert run(budget=-1) == 1
    assert run(q=None) == 1
    assert run(tau=float("nan")) == 1
    assert run(wsb=8) == 7
    assert run(g=mkv.geom(1, 2, 5, 64)) == 2
