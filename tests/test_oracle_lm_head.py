"""Pins of the oracle's LM-head projection (logits = h W^T from bf16 operands, Section 2.1) and of
the verify epilogue built on it, against what the mathematics fixes: one-hot weight rows select
single state entries, a planted direction gives a closed-form logit, the plain product equals
numpy's BLAS matmul, nonnegative operands make the error scale equal the logits, and drafter
states equal to the target's (q = p) accept every draft."""
import numpy as np
import pytest

import oracle
from paper_2606_31315_gb300 import workloads as wl

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


def bits(x):
    return wl.f32_to_bf16_bits(np.asarray(x, dtype=np.float32))


def test_one_hot_rows_select_state_entries():
    """W[v] = c_v e_{pi(v)} (c_v = +-2^j, exact in bf16): logits[r, v] = c_v h[r, pi(v)] exactly.
    A transposed operand, a wrong row or a dropped scale fails this."""
    rng = np.random.default_rng(0)
    V, H, R = 37, 16, 5
    pi = rng.integers(0, H, size=V)
    c = rng.choice([-4.0, -0.5, 0.25, 1.0, 8.0], size=V)
    w = np.zeros((V, H), dtype=np.float32)
    w[np.arange(V), pi] = c
    h = bits(rng.standard_normal((R, H)))
    got = oracle.lm_head_logits(bits(w), h)
    hv = wl.bf16_bits_to_f32(h).astype(np.float64)
    np.testing.assert_array_equal(got, c[None, :] * hv[:, pi])


def test_planted_direction_closed_form():
    """w_d in {+-1}^H and h = 2^-2 w_d: logits[d] = H / 4 exactly; other rows get 2^-2 <w_v, w_d>."""
    rng = np.random.default_rng(1)
    V, H = 20, 64
    w = rng.choice([-1.0, 1.0], size=(V, H)).astype(np.float32)
    h = 0.25 * w[[7, 3]]
    got = oracle.lm_head_logits(bits(w), bits(h))
    assert got[0, 7] == H / 4 and got[1, 3] == H / 4
    np.testing.assert_array_equal(got, 0.25 * (w.astype(np.float64) @ w[[7, 3]].T.astype(np.float64)).T)


def test_equals_blas_matmul_and_error_scale():
    """Random bf16 operands: equal to numpy's fp64 matmul of the widened values (to fp64 rounding,
    measured against the error scale), and the error scale equals |W| |h|^T."""
    rng = np.random.default_rng(2)
    V, H, R = 257, 192, 7
    w, h = bits(rng.standard_normal((V, H)) * 0.1), bits(rng.standard_normal((R, H)))
    got, mag = oracle.lm_head_logits(w, h, with_abs=True)
    wf, hf = wl.bf16_bits_to_f32(w).astype(np.float64), wl.bf16_bits_to_f32(h).astype(np.float64)
    assert np.all(np.abs(got - hf @ wf.T) <= 1e-13 * mag)
    np.testing.assert_allclose(mag, np.abs(hf) @ np.abs(wf).T, rtol=1e-13)
    assert np.all(mag >= np.abs(got))


def test_nonnegative_operands_error_scale_equals_logits():
    rng = np.random.default_rng(3)
    w, h = bits(rng.random((50, 32))), bits(rng.random((3, 32)))
    got, mag = oracle.lm_head_logits(w, h, with_abs=True)
    np.testing.assert_array_equal(got, mag)


def test_linearity_in_the_state():
    """Small-integer states (exact in bf16 and their sum too): logits(h1 + h2) = logits(h1) + logits(h2)."""
    rng = np.random.default_rng(4)
    w = bits(rng.standard_normal((40, 24)))
    h1, h2 = rng.integers(-8, 8, size=(2, 24)), rng.integers(-8, 8, size=(2, 24))
    l1, l2 = oracle.lm_head_logits(w, bits(h1)), oracle.lm_head_logits(w, bits(h2))
    np.testing.assert_allclose(oracle.lm_head_logits(w, bits(h1 + h2)), l1 + l2, rtol=0, atol=1e-12)


def test_drafter_equal_to_target_accepts_every_draft():
    """h_draft = the target row's state gives q = p at every position: a_i = 1 and n_acc = gamma
    for every sequence, whatever the draft tokens; the bonus token follows p_gamma."""
    w = wl.custom(seed=5, ctx=(0, 0, 0), block=(6, 1, 9), vocab=777)
    inp = wl.lm_head_inputs(w, 1.0, hidden=64)
    cu = inp["cu_draft"]
    trow = np.concatenate([np.arange(cu[s], cu[s + 1]) + s for s in range(3)])
    res = oracle.verify_epilogue(inp["w"], inp["h_target"], inp["h_target"][trow], inp["draft_tokens"], cu, 1.0,
                                 inp["u_accept"], inp["u_sample"])
    np.testing.assert_array_equal(res["n_accepted"], np.diff(cu))
    assert np.all(res["accept_prob"] == 1.0)


def test_greedy_epilogue_accepts_target_argmax_drafts():
    """T = 0: drafts equal to the argmax of their target row are all accepted and the bonus token
    is the last row's argmax; the drafter's states are not needed."""
    w = wl.custom(seed=6, ctx=(0, 0), block=(5, 8), vocab=1500)
    inp = wl.lm_head_inputs(w, 0.0, hidden=64)
    cu = inp["cu_draft"]
    tl = oracle.lm_head_logits(inp["w"], inp["h_target"])
    trow = np.concatenate([np.arange(cu[s], cu[s + 1]) + s for s in range(2)])
    tokens = np.argmax(tl[trow], axis=1).astype(np.int32)
    res = oracle.verify_epilogue(inp["w"], inp["h_target"], None, tokens, cu, 0.0)
    np.testing.assert_array_equal(res["n_accepted"], np.diff(cu))
    last = [cu[s + 1] + s for s in range(2)]
    np.testing.assert_array_equal(res["out_tokens"][last], np.argmax(tl[last], axis=1))


def test_workload_plants_the_drafters_boost():
    """The generator's push raises the drafter's logit of its token by `boost` (up to the bf16
    rounding of the state), so drafts sit near the top of the drafter's distribution."""
    w = wl.custom(seed=7, ctx=(0,), block=(12,), vocab=5000)
    inp = wl.lm_head_inputs(w, 1.0, hidden=256, boost=18.0)
    dl = oracle.lm_head_logits(inp["w"], inp["h_draft"])
    x = inp["draft_tokens"]
    at = dl[np.arange(len(x)), x]
    others = np.delete(dl, x, axis=1) if len(set(x)) == len(x) else dl
    # boost + the token's own N(0, 9) base logit + N(0, 1) noise: the mean of 12 is within 3.5 sigma of 18
    assert abs(at.mean() - 18.0) < 3.5 * np.sqrt(10.0 / len(x))
    assert np.median(at) > np.percentile(others, 99.9)
