"""The named synthetic workloads stand for five fixed configurations; these tests pin each one's shapes,
distributions and structure to its stated recipe (CPU only)."""
import numpy as np
import pytest

from paper_2606_31315_gb300 import workloads as wl


def test_candidate_block_sizes():
    np.testing.assert_array_equal(wl.CANDIDATES, np.arange(8, 25, 2))


def test_tiny_fp32():
    w = wl.get("tiny")
    assert (w.num_seqs, w.ctx, w.block, w.num_q_heads, w.num_kv_heads, w.head_dim, w.dtype, w.vocab) == \
        (1, (256,), (8,), 4, 2, 64, "f32", 1024)
    assert w.logit_std == 2.0 and w.temperatures == (1.0,)
    assert w.policy["d_in"] == 1024 and w.policy["hidden"] == 256


def test_qwen3_4b_single_layer_verify():
    w = wl.get("qwen3_4b")
    assert (w.num_seqs, w.ctx, w.block, w.num_q_heads, w.num_kv_heads, w.head_dim, w.dtype, w.vocab) == \
        (1, (2048,), (16,), 32, 8, 128, "bf16", 151936)
    assert set(w.temperatures) == {0.0, 1.0}


def test_ragged_batch_structure():
    w = wl.get("ragged")
    assert w.num_seqs == 32 and len(w.block) == 32 and len(w.ctx) == 32
    assert set(w.block) <= {8, 10, 12, 14, 16, 18, 20, 24}
    assert all(512 <= c <= 8192 for c in w.ctx)
    assert (w.num_q_heads, w.num_kv_heads, w.head_dim, w.vocab) == (32, 8, 128, 151936)
    assert w.policy == dict(num_reqs=32, d_in=2560, hidden=2048, wdtype="bf16", feat_std=1.0)
    # the block sampler itself: 60% of the mass on 14-18, the rest spread over the other five sizes,
    # contexts uniform over [512, 8192] (checked on a large draw from the same generators)
    b = np.array(wl._ragged_blocks(11, 200_000))
    assert abs(np.isin(b, (14, 16, 18)).mean() - 0.6) < 0.005
    for size in (8, 10, 12, 20, 24):
        assert abs((b == size).mean() - 0.08) < 0.003
    c = np.array(wl._ragged_ctx(11, 200_000))
    assert c.min() == 512 and c.max() == 8192
    assert abs(c.mean() - (512 + 8192) / 2) < 20


def test_drafter_and_long_context():
    d = wl.get("drafter_bidir")
    assert (d.num_seqs, d.ctx, d.block, d.mask, d.has_accept) == (16, (4096,) * 16, (16,) * 16, "bidir", False)
    lc = wl.get("long_context")
    assert (lc.num_seqs, lc.ctx, lc.block) == (8, (32768,) * 8, (16,) * 8)
    assert set(lc.temperatures) == {0.0, 1.0}


@pytest.mark.parametrize("temp", [1.0, 0.0])
def test_acceptance_recipe(temp):
    """Target logits ~ N(0, logit_std^2); draft = the matching target row + N(0, 1); T = 1 tokens drawn
    from the drafter (Gumbel-max), T = 0 tokens its argmax; target rows of sequence s start at
    cu_draft[s] + s."""
    w = wl.get("qwen3_4b")
    a = wl.accept_inputs(w, temp)
    t, d = a["target_logits"], a["draft_logits"]
    assert t.shape == (16, 151936) and d.shape == (15, 151936) and t.dtype == np.float32
    assert abs(t.std() - 3.0) < 0.01 and abs(t.mean()) < 0.01
    noise = d.astype(np.float64) - t[:15]
    assert abs(noise.std() - 1.0) < 0.01 and abs(noise.mean()) < 0.01
    np.testing.assert_array_equal(a["cu_draft"], [0, 15])
    tok = a["draft_tokens"]
    if temp == 0.0:
        np.testing.assert_array_equal(tok, np.argmax(d, axis=1))
    else:  # sampled from q: the drafted token is far up the drafter's distribution, not its argmax
        ranks = (d > d[np.arange(15), tok][:, None]).sum(axis=1)
        assert np.median(ranks) < 2000 and not np.array_equal(tok, np.argmax(d, axis=1))
    assert ((a["u_accept"] >= 0) & (a["u_accept"] < 1)).all() and a["u_sample"].shape == (1,)
