"""Helpers for the GPU parity tests: device tensors from numpy arrays, and the
comparison rules.  Tolerances (from the method's error budget):
  decode outputs   max |gpu - oracle| <= 2e-3 * ||o_oracle||_inf per query head
                   (bf16 inputs, fp32 accumulation)
  moments          max |gpu - oracle| <= 1e-4 * max |oracle| per tensor and unit
  index sets       identical wherever the oracle's boundary gap exceeds 1e-5
                   (relative); otherwise only swaps across the near-tie
"""
import numpy as np
import torch

from paper_2606_01563_gb300.inputs import to_bf16_tensor

DECODE_TOL = 2e-3
MOMENT_TOL = 1e-4
GAP_EXACT = 1e-5


def bf16(x):
    return to_bf16_tensor(x).cuda()


def f32(x):
    return torch.from_numpy(np.ascontiguousarray(x, np.float32)).cuda()


def i32(x):
    return torch.from_numpy(np.ascontiguousarray(x, np.int32)).cuda()


def host(t):
    return t.detach().float().cpu().numpy() if t.dtype != torch.int32 else t.cpu().numpy()


def assert_output_close(got, ref, what=""):
    """got, ref: [..., d]; per-row max-abs error within DECODE_TOL * ||ref row||_inf."""
    got = np.asarray(got, np.float64).reshape(-1, got.shape[-1])
    ref = np.asarray(ref, np.float64).reshape(-1, ref.shape[-1])
    assert np.isfinite(got).all(), f"{what}: non-finite output"
    err = np.abs(got - ref).max(axis=1)
    lim = DECODE_TOL * np.abs(ref).max(axis=1)
    bad = np.nonzero(err > lim)[0]
    assert bad.size == 0, f"{what}: rows {bad[:8]} err {err[bad[:8]]} > {lim[bad[:8]]}"


def assert_moment_close(got, ref, what=""):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    scale = max(np.abs(ref).max(), 1e-30)
    err = np.abs(got - ref).max() if ref.size else 0.0
    assert err <= MOMENT_TOL * scale, f"{what}: max err {err:.3e} > {MOMENT_TOL} * {scale:.3e}"
