"""Python binding of the MomentKV C ABI (include/mkv.h).

Argument marshalling only: every function forwards to the function of the
same name in libmkv.so, passing device pointers of torch tensors; all work
runs in the library's CUDA kernels.  A non-OK status raises MKVError.  The
library is loaded on first use and a missing build raises immediately --
there is no fallback implementation.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libmkv.so")

c_i32 = ctypes.c_int32
c_vp = ctypes.c_void_p


class mkv_geom(ctypes.Structure):
    _fields_ = [("batch", c_i32), ("n_kv_heads", c_i32), ("group", c_i32), ("head_dim", c_i32)]


class mkv_moments(ctypes.Structure):
    _fields_ = [("n", c_vp), ("mu_k", c_vp), ("mu_v", c_vp), ("C", c_vp)]


class mkv_cache(ctypes.Structure):
    _fields_ = [("K", c_vp), ("V", c_vp), ("pos", c_vp), ("len", c_vp), ("seen", c_vp), ("capacity", c_i32),
                ("y", c_vp), ("y_len", c_vp)]


class mkv_compress_params(ctypes.Structure):
    _fields_ = [("budget", c_i32), ("window", c_i32), ("sink", c_i32), ("keep_window", c_i32),
                ("pool", c_i32), ("mi", c_i32), ("causal", c_i32), ("tau", ctypes.c_float), ("adaptive", c_i32)]


class mkv_compress_diag(ctypes.Structure):
    _fields_ = [("scores", c_vp), ("score2", c_vp), ("idx_stage1", c_vp)]


class mkv_decode_params(ctypes.Structure):
    _fields_ = [("correction", c_i32), ("order", c_i32), ("tau", ctypes.c_float), ("C16", c_vp),
                ("early_load", c_i32), ("C_split", c_vp)]


STATUS = {0: "MKV_OK", 1: "MKV_ERR_INVALID_ARG", 2: "MKV_ERR_SHAPE", 3: "MKV_ERR_CAPACITY",
          4: "MKV_ERR_CUDA", 5: "MKV_ERR_TIMEOUT", 6: "MKV_ERR_UNSUPPORTED", 7: "MKV_ERR_WORKSPACE"}

EXPORTS = ("mkv_status_str", "mkv_version", "mkv_compress_workspace_size", "mkv_compress",
           "mkv_decode_workspace_size", "mkv_decode_step", "mkv_evict_workspace_size",
           "mkv_evict_append", "mkv_get_device_error", "mkv_decode_step_noalloc", "mkv_moments_pack_bf16",
           "mkv_decode_evict_workspace_size", "mkv_decode_evict_step", "mkv_moments_pack_split")
# test hooks declared in include/mkv_debug.h
DEBUG_EXPORTS = ("mkv_debug_set_poll_limit", "mkv_debug_force_ticket_merge")


class MKVError(RuntimeError):
    def __init__(self, code, where):
        self.code = code
        super().__init__(f"{where}: {STATUS.get(code, code)} ({lib().mkv_status_str(code).decode()})")


_lib = None


def lib():
    """The loaded libmkv.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"{LIB_PATH} is missing: build it first "
                              "(python -c 'import __graft_entry__ as g; g.build()')")
        L = ctypes.CDLL(LIB_PATH)
        L.mkv_status_str.restype = ctypes.c_char_p
        L.mkv_status_str.argtypes = [c_i32]
        L.mkv_version.restype = c_i32
        L.mkv_compress_workspace_size.restype = ctypes.c_size_t
        L.mkv_compress_workspace_size.argtypes = [mkv_geom, c_i32, ctypes.POINTER(mkv_compress_params)]
        L.mkv_compress.restype = c_i32
        L.mkv_compress.argtypes = [mkv_geom, c_i32, c_vp, c_vp, c_vp, ctypes.POINTER(mkv_compress_params),
                                   ctypes.POINTER(mkv_cache), ctypes.POINTER(mkv_moments),
                                   ctypes.POINTER(mkv_compress_diag), c_vp, ctypes.c_size_t, c_vp]
        L.mkv_decode_workspace_size.restype = ctypes.c_size_t
        L.mkv_decode_workspace_size.argtypes = [mkv_geom, c_i32]
        L.mkv_decode_step.restype = c_i32
        L.mkv_decode_step.argtypes = [mkv_geom, c_vp, c_vp, c_vp, ctypes.POINTER(mkv_cache),
                                      ctypes.POINTER(mkv_moments), ctypes.POINTER(mkv_decode_params),
                                      c_vp, c_vp, c_vp, ctypes.c_size_t, c_vp]
        L.mkv_decode_step_noalloc.restype = c_i32
        L.mkv_decode_step_noalloc.argtypes = [mkv_geom, c_vp, c_vp, c_vp, ctypes.POINTER(mkv_cache),
                                              ctypes.POINTER(mkv_moments), ctypes.POINTER(mkv_decode_params),
                                              c_vp, c_vp, c_vp]
        L.mkv_evict_workspace_size.restype = ctypes.c_size_t
        L.mkv_evict_workspace_size.argtypes = [mkv_geom, c_i32]
        L.mkv_evict_append.restype = c_i32
        L.mkv_evict_append.argtypes = [mkv_geom, c_vp, c_vp, c_vp, c_i32, ctypes.POINTER(mkv_cache),
                                       ctypes.POINTER(mkv_moments), ctypes.c_float, c_vp, ctypes.c_size_t, c_vp]
        L.mkv_decode_evict_workspace_size.restype = ctypes.c_size_t
        L.mkv_decode_evict_workspace_size.argtypes = [mkv_geom, c_i32]
        L.mkv_decode_evict_step.restype = c_i32
        L.mkv_decode_evict_step.argtypes = [mkv_geom, c_vp, c_vp, c_vp, c_i32, ctypes.POINTER(mkv_cache),
                                            ctypes.POINTER(mkv_moments), ctypes.POINTER(mkv_decode_params),
                                            c_vp, c_vp, c_vp, ctypes.c_size_t, c_vp]
        L.mkv_moments_pack_bf16.restype = c_i32
        L.mkv_moments_pack_bf16.argtypes = [mkv_geom, ctypes.POINTER(mkv_moments), c_vp, c_vp]
        L.mkv_moments_pack_split.restype = c_i32
        L.mkv_moments_pack_split.argtypes = [mkv_geom, ctypes.POINTER(mkv_moments), ctypes.c_float, c_vp, c_vp]
        L.mkv_debug_set_poll_limit.restype = ctypes.c_int64
        L.mkv_debug_set_poll_limit.argtypes = [ctypes.c_int64]
        L.mkv_debug_force_ticket_merge.restype = c_i32
        L.mkv_debug_force_ticket_merge.argtypes = [c_i32]
        L.mkv_get_device_error.restype = c_i32
        L.mkv_get_device_error.argtypes = [c_vp, c_vp, ctypes.POINTER(c_i32)]
        _lib = L
    return _lib


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _check(code, where):
    if code != 0:
        raise MKVError(code, where)


# ----------------------------------------------------------------- state
@dataclass
class Cache:
    """Retained KV cache (mkv_cache): K, V bf16 [b, h_kv, cap, d]; pos [b, h_kv, cap];
    len, seen [b, h_kv] (int32)."""
    K: torch.Tensor
    V: torch.Tensor
    pos: torch.Tensor
    len: torch.Tensor
    seen: torch.Tensor
    y: torch.Tensor | None = None      # optional eviction state: fp32 [b, h_kv, cap, d]
    y_len: torch.Tensor | None = None  # int32 [b, h_kv]

    @property
    def capacity(self):
        return self.K.shape[2]

    def c(self):
        return mkv_cache(self.K.data_ptr(), self.V.data_ptr(), self.pos.data_ptr(), self.len.data_ptr(),
                         self.seen.data_ptr(), self.capacity, None if self.y is None else self.y.data_ptr(),
                         None if self.y_len is None else self.y_len.data_ptr())


@dataclass
class Moments:
    """Evicted-set moments (mkv_moments): n [b, h_kv] int32; mu_k, mu_v [b, h_kv, d]; C [b, h_kv, d, d]."""
    n: torch.Tensor
    mu_k: torch.Tensor
    mu_v: torch.Tensor
    C: torch.Tensor

    def c(self):
        return mkv_moments(self.n.data_ptr(), self.mu_k.data_ptr(), self.mu_v.data_ptr(), self.C.data_ptr())


def geom(batch, n_kv_heads, group, head_dim):
    return mkv_geom(batch, n_kv_heads, group, head_dim)


def alloc_cache(g: mkv_geom, capacity, device="cuda", evict_state=False):
    """A zero cache; evict_state adds the y rows and y_len of the eviction state."""
    shp = (g.batch, g.n_kv_heads)
    y = torch.zeros(*shp, capacity, g.head_dim, dtype=torch.float32, device=device) if evict_state else None
    y_len = torch.zeros(*shp, dtype=torch.int32, device=device) if evict_state else None
    return Cache(torch.zeros(*shp, capacity, g.head_dim, dtype=torch.bfloat16, device=device),
                 torch.zeros(*shp, capacity, g.head_dim, dtype=torch.bfloat16, device=device),
                 torch.zeros(*shp, capacity, dtype=torch.int32, device=device),
                 torch.zeros(*shp, dtype=torch.int32, device=device),
                 torch.zeros(*shp, dtype=torch.int32, device=device), y, y_len)


def alloc_moments(g: mkv_geom, device="cuda"):
    shp = (g.batch, g.n_kv_heads)
    d = g.head_dim
    return Moments(torch.zeros(*shp, dtype=torch.int32, device=device),
                   torch.zeros(*shp, d, dtype=torch.float32, device=device),
                   torch.zeros(*shp, d, dtype=torch.float32, device=device),
                   torch.zeros(*shp, d, d, dtype=torch.float32, device=device))


def alloc_workspace(nbytes, device="cuda"):
    """Zero-filled device workspace (torch's allocator returns 512-byte aligned blocks)."""
    return torch.zeros(max(int(nbytes), 256), dtype=torch.uint8, device=device)


# ------------------------------------------------------------- functions
def mkv_version():
    return lib().mkv_version()


def mkv_status_str(code):
    return lib().mkv_status_str(code).decode()


def mkv_compress_workspace_size(g, T, p: mkv_compress_params):
    return lib().mkv_compress_workspace_size(g, T, ctypes.byref(p))


def mkv_decode_workspace_size(g, capacity):
    return lib().mkv_decode_workspace_size(g, capacity)


def mkv_evict_workspace_size(g, capacity):
    return lib().mkv_evict_workspace_size(g, capacity)


def mkv_compress(g, T, K, V, Q_obs, p: mkv_compress_params, cache: Cache, mom: Moments, ws, diag=None,
                 stream=None):
    d = mkv_compress_diag(*(None if x is None else x.data_ptr() for x in (diag or (None, None, None))))
    c, m = cache.c(), mom.c()
    code = lib().mkv_compress(g, T, _ptr(K), _ptr(V), _ptr(Q_obs), ctypes.byref(p), ctypes.byref(c),
                              ctypes.byref(m), ctypes.byref(d), _ptr(ws), ws.numel(), _stream(stream))
    _check(code, "mkv_compress")


def mkv_decode_step(g, q, k_new, v_new, cache: Cache, mom: Moments | None, p: mkv_decode_params, out, lse,
                    ws, stream=None):
    c = cache.c()
    m = mom.c() if mom is not None else None
    code = lib().mkv_decode_step(g, _ptr(q), _ptr(k_new), _ptr(v_new), ctypes.byref(c),
                                 ctypes.byref(m) if m is not None else None, ctypes.byref(p), _ptr(out),
                                 _ptr(lse), _ptr(ws), ws.numel(), _stream(stream))
    _check(code, "mkv_decode_step")


def mkv_decode_step_noalloc(g, q, k_new, v_new, cache: Cache, mom: Moments | None, p: mkv_decode_params, out,
                            lse, stream=None):
    """mkv_decode_step with the library's fixed device scratch instead of a workspace."""
    c = cache.c()
    m = mom.c() if mom is not None else None
    code = lib().mkv_decode_step_noalloc(g, _ptr(q), _ptr(k_new), _ptr(v_new), ctypes.byref(c),
                                         ctypes.byref(m) if m is not None else None, ctypes.byref(p), _ptr(out),
                                         _ptr(lse), _stream(stream))
    _check(code, "mkv_decode_step_noalloc")


def mkv_evict_append(g, q, k_new, v_new, budget, cache: Cache, mom: Moments, tau, ws, stream=None):
    c, m = cache.c(), mom.c()
    code = lib().mkv_evict_append(g, _ptr(q), _ptr(k_new), _ptr(v_new), budget, ctypes.byref(c),
                                  ctypes.byref(m), tau, _ptr(ws), ws.numel(), _stream(stream))
    _check(code, "mkv_evict_append")


def mkv_decode_evict_workspace_size(g, capacity):
    return lib().mkv_decode_evict_workspace_size(g, capacity)


def mkv_decode_evict_step(g, q, k_new, v_new, budget, cache: Cache, mom: Moments, p: mkv_decode_params, out, lse,
                          ws, stream=None):
    """Algorithm 1 for one generated token: append, evict down to `budget`, corrected output."""
    c, m = cache.c(), mom.c()
    code = lib().mkv_decode_evict_step(g, _ptr(q), _ptr(k_new), _ptr(v_new), budget, ctypes.byref(c),
                                       ctypes.byref(m), ctypes.byref(p), _ptr(out), _ptr(lse), _ptr(ws), ws.numel(),
                                       _stream(stream))
    _check(code, "mkv_decode_evict_step")


def mkv_moments_pack_bf16(g, mom: Moments, C16, stream=None):
    """C16 (bf16 [b, h_kv, d, d]) = bf16(mom.C): the 16-bit copy mkv_decode_params.C16 points at."""
    m = mom.c()
    _check(lib().mkv_moments_pack_bf16(g, ctypes.byref(m), _ptr(C16), _stream(stream)), "mkv_moments_pack_bf16")


def mkv_moments_pack_split(g, mom: Moments, tau, C_split, stream=None):
    """C_split (int32 [b, h_kv, d, d], as many bytes as C) = the (hi, lo) bf16x2
    operand words of the clamped C': what mkv_decode_params.C_split points at."""
    m = mom.c()
    _check(lib().mkv_moments_pack_split(g, ctypes.byref(m), float(tau), _ptr(C_split), _stream(stream)),
           "mkv_moments_pack_split")


def mkv_debug_set_poll_limit(polls):
    """Test hook (include/mkv_debug.h): poll limit of the kernels' pipeline
    waits; negative restores the default.  Returns the previous limit."""
    return lib().mkv_debug_set_poll_limit(int(polls))


def mkv_debug_force_ticket_merge(on):
    """Test hook (include/mkv_debug.h): decode merges through global partials."""
    return lib().mkv_debug_force_ticket_merge(1 if on else 0)


def mkv_get_device_error(ws, stream=None):
    """(status, info) recorded by kernels in this workspace; clears it."""
    info = c_i32(0)
    code = lib().mkv_get_device_error(_ptr(ws), _stream(stream), ctypes.byref(info))
    return code, info.value
