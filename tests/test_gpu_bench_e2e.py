"""The benchmark's end-to-end leg does the device-timed leg's work.

Each run of the bench holds a second graph set over a second device input set:
the double buffer that the pipelined end-to-end steps alternate between.
Once that set holds the same inputs, its replay must give the first set's
outputs bit for bit (the kernels are deterministic: fixed merge orders,
integer histograms).  The pipelined steps themselves (copies on their own
stream, outputs read back on a third) must leave the same outputs and copy
exactly the bytes they report.  Two layers of the one-layer Llama-3.1-8B
workload (T = 8192), budgets 128 and 512, 64 decode steps each."""
import os
import sys

import pytest
import torch

from paper_2606_01563_gb300 import inputs, mkv

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def test_second_input_set_and_pipelined_steps_match():
    dev = torch.device("cuda", 0)
    wl = inputs.WORKLOADS["llama8b_layer_t8k"]
    stack = bench.Stack(torch, inputs, wl, seed=5, dev=dev, layers=2, steps=64)
    runs = [bench.Run(torch, mkv, stack, B, 0, dev) for B in (128, 512)]
    stream = torch.cuda.Stream(dev)
    for r in runs:
        r.capture(stream)
    bench.replay(runs, stream)
    stream.synchronize()
    for r in runs:
        r.check_errors(stream)
    ref = [r.final.clone() for r in runs]
    assert all(torch.isfinite(f).all() for f in ref)

    twin = stack.twin()
    for r in runs:
        r.capture(stream, twin)
        assert len(r.graph_sets) == 2 and r.graphs is r.graph_sets[0]
    for r in runs:
        r.final.zero_()
    with torch.cuda.stream(stream):
        for r in runs:
            for _, gr in r.graph_sets[1]:
                gr.replay()
    stream.synchronize()
    for r, f in zip(runs, ref):
        assert torch.equal(r.final, f)

    steps = 3
    for r in runs:
        r.final.zero_()
    total, h2d, d2h, copy_ms = bench.e2e_measure(torch, [stack, twin], runs, stream, steps)
    for r in runs:
        r.check_errors(stream)
    assert total > 0 and len(copy_ms) == steps and all(c > 0 for c in copy_ms)
    assert h2d == stack.nbytes()
    assert d2h == sum(r.final.numel() * r.final.element_size() for r in runs)
    for r, f in zip(runs, ref):
        assert torch.equal(r.final, f)
