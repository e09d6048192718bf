"""mkv_decode_step_noalloc: the decode entry point for callers that cannot
allocate device memory (an engine plugin handed only its input and output
buffers, a server whose memory is reserved up front, a path that cannot take
cudaMalloc's device synchronisation).  Its scratch is the library's fixed
device array.  Two calls in a row must match the workspace entry point,
mkv_decode_step, on identical inputs within the decode tolerance, and
oversized geometries must be rejected.  This file is collected last so that
a stop-at-first-failure run has already run every other test."""
import numpy as np
import pytest
import torch

from paper_2606_01563_gb300 import mkv
from paper_2606_01563_gb300.inputs import bf16_round
from gpu_util import assert_output_close, bf16, f32, host, i32

pytestmark = pytest.mark.gpu


def make(rng, b, H, D, cap, lens):
    K = bf16(bf16_round(rng.standard_normal((b, H, cap, D))))
    V = bf16(bf16_round(rng.standard_normal((b, H, cap, D))))
    return lambda: mkv.Cache(K.clone(), V.clone(), i32(np.zeros((b, H, cap))), i32(lens), i32(lens))


def test_noalloc_matches_workspace_entry_point():
    rng = np.random.default_rng(77)
    b, H, G, D, cap = 2, 8, 4, 128, 600
    g = mkv.geom(b, H, G, D)
    lens = rng.integers(100, cap - 4, (b, H)).astype(np.int32)
    fresh = make(rng, b, H, D, cap, lens)
    cache_ws, cache_na = fresh(), fresh()
    mom = mkv.Moments(i32(rng.integers(1, 9000, (b, H))), f32(0.3 * rng.standard_normal((b, H, D))),
                      f32(0.3 * rng.standard_normal((b, H, D))), f32(0.05 * rng.standard_normal((b, H, D, D))))
    p = mkv.mkv_decode_params(1, 1, 1e-6)
    ws = mkv.alloc_workspace(mkv.mkv_decode_workspace_size(g, cap))
    for call in range(2):
        q = bf16(bf16_round(2.0 * rng.standard_normal((b, H * G, D))))
        kn = bf16(bf16_round(rng.standard_normal((b, H, D))))
        vn = bf16(bf16_round(rng.standard_normal((b, H, D))))
        out_ws = torch.empty(b, H * G, D, device="cuda")
        out_na = torch.full((b, H * G, D), float("nan"), device="cuda")
        lse_ws = torch.empty(b, H * G, device="cuda")
        lse_na = torch.empty(b, H * G, device="cuda")
        mkv.mkv_decode_step(g, q, kn, vn, cache_ws, mom, p, out_ws, lse_ws, ws)
        mkv.mkv_decode_step_noalloc(g, q, kn, vn, cache_na, mom, p, out_na, lse_na)
        torch.cuda.synchronize()
        assert_output_close(host(out_na), host(out_ws), f"call {call}")
        np.testing.assert_allclose(host(lse_na), host(lse_ws), rtol=0, atol=1e-4)
        np.testing.assert_array_equal(host(cache_na.len), host(cache_ws.len))
        np.testing.assert_array_equal(host(cache_na.K), host(cache_ws.K))
    assert mkv.mkv_get_device_error(ws)[0] == 0


def test_noalloc_rejects_oversized_geometry():
    g = mkv.geom(1024, 8, 8, 128)  # one partial per query head alone exceeds the 4 MiB scratch
    cache = mkv.alloc_cache(mkv.geom(1, 1, 1, 128), 4)
    p = mkv.mkv_decode_params(0, 1, 0.0)
    out = torch.empty(1, device="cuda")
    with pytest.raises(mkv.MKVError) as e:
        mkv.mkv_decode_step_noalloc(g, out, None, None, cache, None, p, out, None)
    assert e.value.code == 7
