"""GPU parity of bp_policy_select against the fp64 oracle.

Bars: logits within 1e-3 relative to max |o| (fp32 accumulation of bf16/fp32 products); the
selected block size exact unless the oracle's top-2 margin is below 1e-4 * max |o|.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2606_31315_gb300 as bp
from paper_2606_31315_gb300 import workloads as wl

from _gpu import to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    bp.build()
    bp.load()


def _run(pin):
    dt = "bf16" if pin["wdtype"] == "bf16" else None
    f = lambda k: to_dev(pin[k], dt if k in ("feats", "w1", "w2") else None)  # noqa: E731
    ri = to_dev(pin["row_index"]) if pin.get("row_index") is not None else None
    bs, lo = bp.policy_select(f("feats"), f("w1"), f("b1"), f("w2"), f("b2"), f("candidates"), row_index=ri)
    return bs.cpu().numpy(), lo.cpu().numpy()


def _oracle(pin):
    d = pin["wdtype"]
    return oracle.policy_select(wl.as_f64(pin["feats"], d), wl.as_f64(pin["w1"], d), pin["b1"],
                                wl.as_f64(pin["w2"], d), pin["b2"], pin["candidates"], row_index=pin.get("row_index"))


def _compare(pin):
    bs, lo = _run(pin)
    ref = _oracle(pin)
    scale = np.abs(ref["logits"]).max()
    assert np.abs(lo - ref["logits"]).max() <= 1e-3 * scale
    ok = ref["top2_margin"] >= 1e-4 * scale
    np.testing.assert_array_equal(bs[ok], ref["block_size"][ok])


def test_tiny_fp32():
    _compare(wl.policy_inputs(wl.get("tiny")))


def test_ragged_bf16_32_requests():
    _compare(wl.policy_inputs(wl.get("ragged")))


def test_more_requests_than_one_group():
    w = wl.custom(seed=5, policy=dict(num_reqs=70, d_in=512, hidden=300, wdtype="bf16", feat_std=1.0))
    _compare(wl.policy_inputs(w))


def test_ties_choose_lowest_index():
    pin = wl.policy_inputs(wl.get("tiny"))
    pin["w2"] = np.zeros_like(pin["w2"])
    pin["b2"] = np.array([0, 1, 3, 2, 3, 3, 0, 1, 3], dtype=np.float32)
    bs, _ = _run(pin)
    assert np.all(bs == pin["candidates"][2])


def test_paper_input_width_streams_w1():
    # Section 3.1 feeds the predictor the last-token logit vector, so d_in = V = 151936: far more
    # 64-column W1 atoms per CTA than fit in shared memory at once, so they stream through a ring.
    w = wl.custom(seed=6, policy=dict(num_reqs=4, d_in=151936, hidden=256, wdtype="bf16", feat_std=3.0))
    _compare(wl.policy_inputs(w))


@pytest.mark.parametrize("d_in", [4104, 5160])
def test_d_in_tail_and_two_request_groups(d_in):
    # d_in is not a multiple of 64 (the last atom is zero-filled), 70 requests span two groups of 64
    # (the second only partly filled) and hidden = 300 leaves the last W1 tile partial.  Split over
    # 9 CTAs per tile, d_in = 4104 (65 atoms, 8 per CTA) is loaded at once; d_in = 5160 (81 atoms, 9
    # per CTA) streams through the ring and wraps around it.
    w = wl.custom(seed=7, policy=dict(num_reqs=70, d_in=d_in, hidden=300, wdtype="bf16", feat_std=1.0))
    _compare(wl.policy_inputs(w))
