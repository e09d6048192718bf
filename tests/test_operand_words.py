"""The reference the GPU tests hold the packed operand form of C' to
(tests/test_gpu_decode_split.py), checked on the CPU: hand-worked words for a
few pairs (bf16 bit patterns, first value of a pair in the low half), the
clamp of App. C.2 (|n C_ab| < tau -> 0, both words zero), and hi + lo
recovering each value to about 16 significant bits."""
import numpy as np
import torch

from test_gpu_decode_split import reference_words


def test_hand_worked_pairs():
    C = torch.tensor([1.0, -3.140625, 1e-9, 0.1, 0.0, -2.0 ** -20]).reshape(1, 1, 1, 6).expand(1, 1, 6, 6).clone()
    n = torch.tensor([[10]], dtype=torch.int32)
    w = reference_words(C, n, 1e-6)[0, 0, 0]            # row 0: three pairs x (hi, lo)
    got = [[int(v) for v in pair] for pair in w]
    # 1.0 = 0x3f80 and -3.140625 = 0xc049 are exact in bf16: lo is zero
    assert got[0] == [0xc0493f80, 0]
    # 1e-9 * 10 < 1e-6 is clamped; 0.1 rounds to 0x3dcd (0.10009765625), and
    # the rest, -9.765625e-05, is 0xb8cd
    assert got[1] == [0x3dcd0000, 0xb8cd0000]
    # 0 stays 0; 10 * 2^-20 is above the clamp and exact in bf16 (0xb580)
    assert got[2] == [0xb5800000, 0]


def _halves_to_float(words):
    lo16 = (words & 0xFFFF).to(torch.int32)
    hi16 = ((words >> 16) & 0xFFFF).to(torch.int32)
    to_f = lambda h: (h << 16).view(torch.float32)
    return to_f(lo16), to_f(hi16)


def test_clamp_and_recovery():
    rng = np.random.default_rng(3)
    b, H, D = 1, 2, 8
    C = torch.tensor(rng.standard_normal((b, H, D, D)) * 0.05, dtype=torch.float32)
    C.view(-1)[::7] *= 1e-6                              # entries below the clamp for these counts
    n = torch.tensor([[40, 3000]], dtype=torch.int32)
    tau = 1e-4
    w = reference_words(C, n, tau)                       # [b, H, D, D/2, 2]
    hi_a, hi_b = _halves_to_float(w[..., 0])
    lo_a, lo_b = _halves_to_float(w[..., 1])
    x = torch.stack([hi_a + lo_a, hi_b + lo_b], dim=-1).reshape(b, H, D, D)
    clamped = (C * n.float()[..., None, None]).abs() < tau
    assert clamped.any() and (~clamped).any()
    assert torch.all(x[clamped] == 0)
    keep = ~clamped
    err = (x[keep] - C[keep]).abs() / C[keep].abs()
    assert float(err.max()) < 2.0 ** -15
