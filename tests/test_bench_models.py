"""Host logic of bench.py on CPU: the byte models behind the roofline and step fractions, for
each gate mode and sync pattern, and the flat gradient buffer the gated runs copy into."""
import os
import sys

import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
import workloads as wl  # noqa: E402


def _mn(w):
    return sum(m * n for m, n in w.shapes)


@pytest.fixture(scope="module")
def stack():
    return wl.WORKLOADS["gpt1p3b_stack_r512"]


def test_step_bytes_per_element(stack):
    """bf16 G, tensor-core mode: 28 B/element when every layer syncs in DION_GATE_ALWAYS (fused
    buffer + B Q 8, Bh read of B^T P 2, update 18); in a gated mode 34 on a synced layer (norms
    pass 10, fused B Q reading B from M 6, Bh 2, update 16) and 20 on a local one (norms 10, local
    10); the compulsory floor is 18 either way."""
    mn, L = _mn(stack), stack.num_layers
    planned, compulsory = bench.step_bytes(stack, "bf16")
    assert planned == 28 * mn and compulsory == 18 * mn
    assert bench.step_bytes(stack, "bf16", "per_layer", [1.0] * L)[0] == 34 * mn
    assert bench.step_bytes(stack, "bf16", "global", [0.0] * L)[0] == 20 * mn
    half = bench.step_bytes(stack, "bf16", "per_layer", [0.5] * L)[0]
    assert half == pytest.approx(27 * mn)
    assert bench.step_bytes(stack, "bf16", "global", [0.0] * L)[1] == compulsory


def test_kernel_bytes_follow_branches(stack):
    mn, L = _mn(stack), stack.num_layers
    assert bench.kernel_work("norms_gate", stack, "bf16", "global", [0.0] * L) == ("hbm", 10 * mn, "B")
    assert bench.kernel_work("local", stack, "bf16", "global", [0.0] * L)[1] == 10 * mn
    assert bench.kernel_work("local", stack, "bf16")[1] == 0
    # the update reads G only when B is formed there (DION_GATE_ALWAYS)
    assert bench.kernel_work("tc_update", stack, "bf16")[1] == 18 * mn
    assert bench.kernel_work("tc_update", stack, "bf16", "per_layer", [1.0] * L)[1] == 16 * mn
    assert bench.kernel_work("tc_update", stack, "bf16", "per_layer", [0.25] * L)[1] == pytest.approx(4 * mn)
    # the fused kernel: reads M and G, writes Bh (+ P, P^T); in a gated mode it reads B from M
    mr = sum(m * r for (m, n), r in zip(stack.shapes, stack.ranks()))
    assert bench.kernel_work("tc_form_bq", stack, "bf16")[1] == 8 * mn + 8 * mr
    assert bench.kernel_work("tc_form_bq", stack, "bf16", "global", [1.0] * L)[1] == 6 * mn + 8 * mr
    # per-layer weights count each layer's own work
    wt = [1.0 if l % 6 == 5 else 0.0 for l in range(L)]  # only the 8192 x 2048 layers sync
    big = sum(m * n for l, (m, n) in enumerate(stack.shapes) if l % 6 == 5)
    assert bench.kernel_work("tc_update", stack, "bf16", "per_layer", wt)[1] == 16 * big


def test_bf16x3_gated_splits_b_after_the_gate():
    """BF16X3 with bf16 G: in DION_GATE_ALWAYS the buffer pass writes B and both halves (14 B per
    element); in a gated mode it writes B alone (10) and split_b writes the halves of the syncing
    layers (8 per synced element): 10 per element on a local step, 42 on a synced one."""
    w = wl.WORKLOADS["gpt350m_gate_stress_r256"]
    mn, L = _mn(w), w.num_layers
    assert bench.kernel_work("form_b", w, "bf16x3")[1] == 14 * mn
    assert bench.kernel_work("form_b", w, "bf16x3", "per_layer", [0.0] * L)[1] == 10 * mn
    assert bench.kernel_work("split_b", w, "bf16x3", "per_layer", [0.0] * L)[1] == 0
    assert bench.kernel_work("split_b", w, "bf16x3", "per_layer", [1.0] * L)[1] == 8 * mn
    assert bench.kernel_work("split_b", w, "bf16x3")[0] == "latency"  # returns at once in ALWAYS
    assert bench.step_bytes(w, "bf16x3")[0] == 14 * mn + 24 * mn
    assert bench.step_bytes(w, "bf16x3", "per_layer", [1.0] * L)[0] == 10 * mn + 32 * mn
    assert bench.step_bytes(w, "bf16x3", "per_layer", [0.0] * L)[0] == 10 * mn + 10 * mn


def test_flat_gradient_views_match_layers():
    w = wl.WORKLOADS["gpt160m_block_r192"]
    seq = bench.make_gradient_sequence(wl, w, torch.bfloat16, "cpu", range(3, 5))
    assert len(seq) == 2 and seq[0].numel() == _mn(w)
    views = bench.layer_views(seq[1], w)
    for l, (m, n) in enumerate(w.shapes):
        assert views[l].shape == (m, n) and views[l].is_contiguous()
        assert torch.equal(views[l], wl.gradient(w, l, 4, "cpu").to(torch.bfloat16))
        # 16-byte aligned rows for the plan: every layer starts on a 16-byte boundary
        assert (views[l].data_ptr() - seq[1].data_ptr()) % 16 == 0
