"""The operand form of C' (mkv_moments_pack_split, mkv_decode_params.C_split).

The pack writes, for every column pair of C, the bf16x2 hi and lo words of
the clamped pair (Eq. fused's clamp of App. C.2: |n C_ab| < tau -> 0).  They
are checked bit for bit against torch's own round-to-nearest-even bf16
conversion of the clamped values.  A decode step that reads them must then
give exactly the output and lse of the step that clamps and splits C itself.
Both decode kernels are covered: the cluster kernel, and the ticket kernel
through its test switch.  The fp32-C path is compared with the fp64 oracle
in test_gpu_decode.py, so bit equality carries that parity over."""
import numpy as np
import pytest
import torch

from paper_2606_01563_gb300 import mkv
from gpu_util import bf16, f32, i32
from test_gpu_decode import make_state

pytestmark = pytest.mark.gpu


def reference_words(C, n, tau):
    """(hi, lo) words per column pair, as int64 [b, h, d, d/2, 2] holding 32 bits."""
    x = C.float()
    x = torch.where((x * n.float()[..., None, None]).abs() < tau, torch.zeros_like(x), x)
    hi = x.to(torch.bfloat16)
    lo = (x - hi.float()).to(torch.bfloat16)
    h16 = hi.view(torch.int16).to(torch.int64) & 0xFFFF
    l16 = lo.view(torch.int16).to(torch.int64) & 0xFFFF
    b, H, D, _ = C.shape
    hw = h16.reshape(b, H, D, D // 2, 2)
    lw = l16.reshape(b, H, D, D // 2, 2)
    # the first value of a pair in the low half
    return torch.stack([hw[..., 0] | (hw[..., 1] << 16), lw[..., 0] | (lw[..., 1] << 16)], dim=-1)


CASES = [
    # b, H, G, D, lens, cap, n_list, tau, early, ticket
    (1, 2, 2, 64, [100, 37], 160, [50, 3], 1e-6, 0, 0),
    (2, 8, 4, 128, None, 640, None, 1e-6, 1, 0),
    (2, 8, 4, 128, None, 640, None, 1e-6, 0, 1),
    (1, 4, 8, 128, [513, 1, 32, 33], 600, [10, 0, 1, 1000], 0.5, 0, 0),
    (1, 4, 8, 128, [513, 1, 32, 33], 600, [10, 0, 1, 1000], 0.5, 0, 1),
    (3, 2, 1, 64, [31, 64, 65, 200, 7, 129], 256, [0, 5, 9, 100, 2, 40], 0.05, 1, 0),
    (4, 8, 4, 128, None, 1340, None, 1e-6, 1, 0),
]


@pytest.mark.parametrize("case", range(len(CASES)))
@pytest.mark.parametrize("new", [False, True])
def test_operand_form_matches_fp32_c(case, new):
    b, H, G, D, lens, cap, n_list, tau, early, ticket = CASES[case]
    rng = np.random.default_rng(900 + case)
    units = b * H
    if lens is None:
        lens = rng.integers(1, cap - 1, units).tolist()
    if n_list is None:
        n_list = rng.integers(0, 4000, units).tolist()
    st = make_state(rng, b, H, G, D, lens, cap, n_list)
    C = st["C"].copy()
    C.reshape(-1)[::97] = 0.0                            # exact zeros stay zero
    C.reshape(-1)[5::89] *= 1e-4                         # entries the larger tau clamps
    g = mkv.geom(b, H, G, D)
    mom = mkv.Moments(i32(st["n"]), f32(st["mu_k"]), f32(st["mu_v"]), f32(C))

    words = torch.empty(b, H, D, D, dtype=torch.int32, device="cuda")
    mkv.mkv_moments_pack_split(g, mom, tau, words)
    torch.cuda.synchronize()
    ref = reference_words(mom.C, mom.n, tau)
    assert torch.equal(words.view(b, H, D, D // 2, 2).to(torch.int64) & 0xFFFFFFFF, ref)

    outs = []
    prev = mkv.mkv_debug_force_ticket_merge(ticket)
    try:
        for split in (None, words):
            cache = mkv.Cache(bf16(st["K"]), bf16(st["V"]),
                              i32(np.broadcast_to(np.arange(cap), (b, H, cap))),
                              i32(st["lens"]), i32(st["lens"] + 1000))
            out = torch.empty(b, H * G, D, device="cuda")
            lse = torch.empty(b, H * G, device="cuda")
            ws = mkv.alloc_workspace(mkv.mkv_decode_workspace_size(g, cap))
            p = mkv.mkv_decode_params(1, 1, tau, None, early, None if split is None else split.data_ptr())
            kn = bf16(st["kn"]) if new else None
            vn = bf16(st["vn"]) if new else None
            mkv.mkv_decode_step(g, bf16(st["q"]), kn, vn, cache, mom, p, out, lse, ws)
            code, info = mkv.mkv_get_device_error(ws)
            assert code == 0, (code, info)
            outs.append((out, lse, cache.len.clone()))
    finally:
        mkv.mkv_debug_force_ticket_merge(prev)
    (o0, l0, n0), (o1, l1, n1) = outs
    assert torch.isfinite(o0).all()
    assert torch.equal(o0, o1)
    assert torch.equal(l0, l1)
    assert torch.equal(n0, n1)
