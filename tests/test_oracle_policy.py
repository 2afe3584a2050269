"""Pins for the oracle's block-size policy head (CPU only).

Section 2.4 fixes B_hat = argmax_b f(p(x))_b over the candidate set; Section 3.1 fixes a
two-layer MLP of hidden width 2048 (Table 1 gives its size).  Pinned by:
  * special cases: W2 = 0 and b2 = e_c selects candidate c; equal top logits pick the
    lowest index; a strongly negative b1 switches every hidden unit off (ReLU), leaving b2;
  * a one-hot input e_j with identity W2 reads column j of W1 through the activation,
    which catches a transposed W1 or W2;
  * invariants: permuting hidden units leaves the logits unchanged; with zero biases the
    head is positively homogeneous, f(c x) = c f(x) for c > 0, but not odd;
  * pooling: gathering rows by index equals pre-gathered rows;
  * Table 1: a two-layer head at the paper's shape (vocabulary-sized input, hidden 2048,
    2k + 1 = 5 classes) holds 0.31 billion parameters, 0.62 GB in bf16.
"""
import os

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_tau.txt")


def _net(seed, d_in=12, hidden=7, c=5, n=6):
    rng = np.random.default_rng(seed)
    return dict(feats=rng.standard_normal((n, d_in)), w1=rng.standard_normal((hidden, d_in)),
                b1=rng.standard_normal(hidden) * 0.1, w2=rng.standard_normal((c, hidden)),
                b2=rng.standard_normal(c) * 0.1, candidates=np.arange(14, 14 + c, dtype=np.int32))


def _call(oracle_mod, n, **kw):
    return oracle_mod.policy_select(n["feats"], n["w1"], n["b1"], n["w2"], n["b2"], n["candidates"], **kw)


def test_zero_w2_selects_bias_class(oracle_mod):
    n = _net(1)
    n["w2"][:] = 0
    for c in range(5):
        n["b2"] = np.zeros(5)
        n["b2"][c] = 1.0
        res = _call(oracle_mod, n)
        assert np.all(res["block_size"] == n["candidates"][c])


def test_ties_pick_lowest_index(oracle_mod):
    n = _net(2)
    n["w2"][:] = 0
    n["b2"] = np.array([0.0, 2.0, 1.0, 2.0, 2.0])
    res = _call(oracle_mod, n)
    assert np.all(res["block_size"] == n["candidates"][1])
    assert np.all(res["top2_margin"] == 0.0)


def test_relu_switches_units_off(oracle_mod):
    n = _net(3)
    n["b1"][:] = -1e6
    res = _call(oracle_mod, n)
    np.testing.assert_array_equal(res["logits"], np.tile(n["b2"], (6, 1)))


def test_one_hot_input_reads_w1_column(oracle_mod):
    d_in, hidden = 9, 6
    n = _net(4, d_in=d_in, hidden=hidden, c=hidden, n=d_in)
    n["feats"] = np.eye(d_in)
    n["b1"][:] = 0
    n["w2"] = np.eye(hidden)
    n["b2"][:] = 0
    res = _call(oracle_mod, n)
    # logits of request j = relu(W1[:, j])
    np.testing.assert_array_equal(res["logits"], np.maximum(n["w1"].T, 0))


def test_hidden_permutation_invariance(oracle_mod):
    n = _net(5, hidden=11)
    perm = np.random.default_rng(0).permutation(11)
    a = _call(oracle_mod, n)
    n2 = dict(n, w1=n["w1"][perm], b1=n["b1"][perm], w2=n["w2"][:, perm])
    b = _call(oracle_mod, n2)
    np.testing.assert_allclose(a["logits"], b["logits"], rtol=0, atol=1e-13)
    np.testing.assert_array_equal(a["block_size"], b["block_size"])


def test_positive_homogeneity(oracle_mod):
    n = _net(6)
    n["b1"][:] = 0
    n["b2"][:] = 0
    a = _call(oracle_mod, n)
    b = _call(oracle_mod, dict(n, feats=3.0 * n["feats"]))
    np.testing.assert_allclose(b["logits"], 3.0 * a["logits"], rtol=1e-13, atol=1e-13)
    c = _call(oracle_mod, dict(n, feats=-n["feats"]))
    assert np.abs(c["logits"] + a["logits"]).max() > 1e-3  # ReLU: not odd


def test_pooling_gathers_rows(oracle_mod):
    n = _net(7, n=10)
    idx = np.array([9, 0, 3, 3], dtype=np.int32)
    a = _call(oracle_mod, n, row_index=idx)
    b = _call(oracle_mod, dict(n, feats=n["feats"][idx]))
    np.testing.assert_array_equal(a["logits"], b["logits"])
    np.testing.assert_array_equal(a["block_size"], b["block_size"])


def test_table1_size_of_two_layer_head():
    vals = {}
    with open(GOLDEN) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                k, v = line.split()[:2]
                vals[k] = float(v)
    d_in = 151936  # Qwen3 vocabulary: the input is the last token's full predictive distribution (Section 2.2)
    hidden = int(vals["predictor_hidden"])
    classes = 2 * int(vals["radius_k"]) + 1
    params = d_in * hidden + hidden + hidden * classes + classes
    assert round(params * 2 / 1e9, 2) == vals["predictor_param_gb"]
    assert abs(params / 1e9 - vals["predictor_params_b"]) < 0.015


def test_rejects_bad_arguments(oracle_mod):
    n = _net(8)
    with pytest.raises(ValueError):
        _call(oracle_mod, n, row_index=np.array([-1], dtype=np.int32))
