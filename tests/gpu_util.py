"""Helpers for the GPU parity tests: device tensors from numpy arrays, and the
comparison rules.  Tolerances (from the method's error budget):
  decode outputs   max |gpu - oracle| <= 2e-3 * ||o_oracle||_inf per query head
                   (bf16 inputs, fp32 accumulation)
  moments          per element |gpu - oracle| <= 1e-4 * |oracle| + 1e-5 * max |oracle|
                   (1e-4 relative, with an absolute floor 10x below it at the
                   tensor's scale for entries near zero, whose fp32 sums over
                   many tokens carry rounding of the larger terms)
  index sets       identical wherever the oracle's boundary gap exceeds 1e-5
                   (relative); otherwise only swaps across the near-tie
"""
import numpy as np
import torch

from paper_2606_01563_gb300.inputs import to_bf16_tensor

DECODE_TOL = 2e-3
MOMENT_TOL = 1e-4
MOMENT_FLOOR = 1e-5
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
    """Per element: |got - ref| <= MOMENT_TOL * |ref| + MOMENT_FLOOR * max |ref|."""
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    if not ref.size:
        return
    scale = max(np.abs(ref).max(), 1e-30)
    err = np.abs(got - ref)
    lim = MOMENT_TOL * np.abs(ref) + MOMENT_FLOOR * scale
    bad = np.argwhere(err > lim)
    if bad.size:
        i = tuple(bad[np.argmax((err - lim)[tuple(bad.T)])])
        need = float(((err - MOMENT_TOL * np.abs(ref)) / scale).max())
        raise AssertionError(f"{what}: {len(bad)} elements out of tolerance; worst at {i}: got {got[i]:.6e} "
                             f"ref {ref[i]:.6e} (floor needed {need:.2e} of max {scale:.3e})")
