"""GPU parity of bp_spec_accept against the fp64 oracle.

Small problems run on the cluster kernel, large ones (by logits read) on the throughput kernels; the
edge cases below are taken on both sides of that line (blocks_for picks the blocks for either side).

Bars: accept_prob within 1e-5 absolute at every drafted position; n_accepted and the emitted
tokens bit-exact for every sequence not flagged as a near-tie (|u_i - a_i| < 1e-5 at a tested
position, or an inverse-CDF threshold within 1e-5 of a cumulative boundary); greedy (T = 0)
bit-exact with no flags.  Full-size workloads run exactly as the benchmark launches them.
"""
import numpy as np
import pytest
import torch
from scipy import stats

import paper_2606_31315_gb300 as bp
from paper_2606_31315_gb300 import workloads as wl

from _gpu import accept_uses_batch, blocks_for, compare_accept, run_accept, run_oracle_accept, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    bp.build()
    bp.load()


def test_tiny():
    w = wl.get("tiny")
    compare_accept(wl.accept_inputs(w, 1.0), 1.0)


@pytest.mark.parametrize("temp", [1.0, 0.0])
def test_qwen3_4b_full(temp):
    w = wl.get("qwen3_4b")
    compare_accept(wl.accept_inputs(w, temp), temp)


def test_named_workloads_take_the_intended_path():
    for name, temp, batch in (("qwen3_4b", 1.0, False), ("qwen3_4b", 0.0, False), ("tiny", 1.0, False),
                              ("ragged", 1.0, True), ("ragged", 0.0, True), ("long_context", 1.0, True)):
        w = wl.get(name)
        assert accept_uses_batch(tuple(w.block), w.vocab, temp) == batch, name


@pytest.mark.parametrize("temp", [1.0, 0.0])
def test_ragged_batch_full(temp):
    w = wl.get("ragged")
    flagged, s = compare_accept(wl.accept_inputs(w, temp), temp)
    # about a quarter of the draws over a 151936-token vocabulary land within 1e-5 of a CDF
    # boundary (most tokens carry less mass than that); those are checked for validity instead
    assert flagged < s // 2


@pytest.mark.parametrize("temp", [0.0, 1.0])
def test_long_context_full(temp):
    w = wl.get("long_context")
    compare_accept(wl.accept_inputs(w, temp), temp)


@pytest.mark.parametrize("temp", [1.0, 0.0])
def test_planted_long_prefixes(temp):
    """Draft rows copied from target rows with probability 0.9: long accepted prefixes and bonus draws."""
    w = wl.custom(seed=44, ctx=(0,) * 12, block=(16, 16, 8, 24, 1, 16, 16, 12, 16, 20, 16, 2), vocab=151936)
    inp = wl.accept_inputs(w, temp, planted_match=0.9)
    compare_accept(inp, temp)
    n_acc, _, _, _ = run_accept(inp, temp)
    assert n_acc.max() >= 10


@pytest.mark.parametrize("temp", [1.0, 0.0])
def test_blocks_longer_than_a_warp_batch(temp):
    """Blocks of up to 64 positions on the throughput kernels, drafts mostly copies of their target rows:
    first rejections past the first 32 positions (the decisions take positions 32 at a time) and bonus
    draws after 63 accepted drafts."""
    blocks = (64, 40, 33, 1, 64, 2) * 3
    assert accept_uses_batch(blocks, 32000, temp)
    w = wl.custom(seed=47, ctx=(0,) * len(blocks), block=blocks, vocab=32000)
    inp = wl.accept_inputs(w, temp, planted_match=0.97)
    compare_accept(inp, temp)
    n_acc, _, _, _ = run_accept(inp, temp)
    assert n_acc.max() > 32


@pytest.mark.parametrize("temp", [1.0, 0.0])
@pytest.mark.parametrize("num_seqs", [1, 255, 256])
def test_one_long_or_many_short_sequences(num_seqs, temp):
    """The throughput kernels on one 48-position block over the full vocabulary (the draw's parts all
    belong to one sequence) and on hundreds of 1-4 position blocks (one decision warp and one draw per
    sequence, most of them bonus draws or first-position rejections), against the oracle."""
    rng = np.random.default_rng(num_seqs)
    blocks = (48,) if num_seqs == 1 else tuple(int(x) for x in rng.integers(1, 5, num_seqs))
    vocab = 151936 if num_seqs == 1 else 32000
    assert accept_uses_batch(blocks, vocab, temp)
    w = wl.custom(seed=num_seqs + 3, ctx=(0,) * len(blocks), block=blocks, vocab=vocab)
    compare_accept(wl.accept_inputs(w, temp, planted_match=0.5), temp)


@pytest.mark.parametrize("batch", [False, True])
@pytest.mark.parametrize("vocab", [5, 1001, 4099, 16384, 32000, 50001])
def test_vocab_sizes_and_scalar_path(vocab, batch):
    """Vocabularies below one chunk, exactly one, and ragged last chunks; odd sizes take the scalar loads."""
    for temp in (1.0, 0.0):
        blocks = blocks_for(vocab, temp, batch)
        w = wl.custom(seed=vocab, ctx=(0,) * len(blocks), block=blocks, vocab=vocab)
        compare_accept(wl.accept_inputs(w, temp), temp)


@pytest.mark.parametrize("temp", [0.05, 0.7, 3.0])
def test_temperatures(temp):
    w = wl.custom(seed=int(temp * 100), ctx=(0,) * 10, block=(16,) * 10, vocab=20000)
    compare_accept(wl.accept_inputs(w, temp), temp)


def test_workspace_reuse_gives_identical_results():
    w = wl.custom(seed=9, ctx=(0,) * 5, block=(16, 4, 1, 16, 8), vocab=50000)
    inp = wl.accept_inputs(w, 1.0)
    ws = bp.workspace(bp.spec_accept_workspace_size(5, int(inp["cu_draft"][-1]), 50000), torch.device("cuda"))
    r1 = run_accept(inp, 1.0, ws=ws)
    r2 = run_accept(inp, 1.0, ws=ws)
    for x, y in zip(r1[:3], r2[:3]):
        np.testing.assert_array_equal(x, y)
    compare_accept(inp, 1.0, gpu=r2)


def test_lossless_chi_square_on_gpu():
    """V = 16, gamma = 3, drafts sampled from q: the first emitted token follows p_0 (chi-square at
    alpha = 1e-3 over 2e5 seeded trials), and the GPU agrees with the oracle trial by trial."""
    V, gamma, n = 16, 3, 200_000
    rng = np.random.default_rng(77)
    p_rows = rng.dirichlet(np.full(V, 2.0), size=gamma + 1)
    q_rows = rng.dirichlet(np.full(V, 2.0), size=gamma)
    tl, dl = np.log(p_rows).astype(np.float32), np.log(q_rows).astype(np.float32)
    cdf = np.cumsum(q_rows, axis=1)
    uu = rng.random((n, gamma))
    toks = np.stack([np.minimum(np.searchsorted(cdf[i], uu[:, i], side="right"), V - 1) for i in range(gamma)],
                    axis=1).astype(np.int32)
    inp = dict(target_logits=np.tile(tl, (n, 1)), draft_logits=np.tile(dl, (n, 1)), draft_tokens=toks.reshape(-1),
               cu_draft=(np.arange(n + 1) * gamma).astype(np.int32),
               u_accept=rng.random(n * gamma, dtype=np.float32), u_sample=rng.random(n, dtype=np.float32))
    gpu = run_accept(inp, 1.0)
    n_acc, out = gpu[0], gpu[1].reshape(n, gamma + 1)
    counts = np.bincount(out[:, 0], minlength=V)
    p0 = np.exp(tl[0].astype(np.float64))
    p0 /= p0.sum()
    stat = ((counts - n * p0) ** 2 / (n * p0)).sum()
    assert stat < stats.chi2.ppf(1 - 1e-3, V - 1), stat
    # prefix survival (Appendix A.1): E[n_acc] = sum_i prod_{j<=i} alpha_j
    q = np.exp(dl.astype(np.float64))
    q /= q.sum(axis=1, keepdims=True)
    p = np.exp(tl.astype(np.float64))
    p /= p.sum(axis=1, keepdims=True)
    expect = np.cumprod(np.minimum(p[:gamma], q).sum(axis=1)).sum()
    assert abs(n_acc.mean() - expect) < 5 * n_acc.std() / np.sqrt(n)
    m = 20_000  # trial-by-trial agreement with the oracle on the first m trials
    small = dict(target_logits=inp["target_logits"][: m * (gamma + 1)], draft_logits=inp["draft_logits"][: m * gamma],
                 draft_tokens=inp["draft_tokens"][: m * gamma], cu_draft=inp["cu_draft"][: m + 1],
                 u_accept=inp["u_accept"][: m * gamma], u_sample=inp["u_sample"][:m])
    compare_accept(small, 1.0, gpu=(gpu[0][:m], gpu[1][: m * (gamma + 1)], gpu[2][: m * gamma], 0),
                   ref=run_oracle_accept(small, 1.0))


@pytest.mark.parametrize("batch", [False, True])
def test_out_of_range_draft_token_sets_device_flag(batch):
    blocks = blocks_for(1000, 1.0, batch)
    w = wl.custom(seed=3, ctx=(0,) * len(blocks), block=blocks, vocab=1000)
    inp = wl.accept_inputs(w, 1.0)
    inp["draft_tokens"][2] = 1000  # caught by the kernel's own bounds check, never dereferenced
    status = run_accept(inp, 1.0)[3]
    assert status == 6  # BP_ERR_DEVICE_FLAG


def test_host_side_validation():
    t = torch.zeros((2, 100), device="cuda")
    tok = torch.zeros(1, dtype=torch.int32, device="cuda")
    cu = torch.tensor([0, 1], dtype=torch.int32, device="cuda")
    with pytest.raises(bp.BlockPilotError) as e:
        bp.spec_accept(t, None, tok, cu, 1.0, torch.zeros(1, device="cuda"), torch.zeros(1, device="cuda"))
    assert e.value.status == 1  # T > 0 needs draft logits


@pytest.mark.parametrize("batch", [False, True])
@pytest.mark.parametrize("temp", [1.0, 0.0])
def test_masked_vocabulary(temp, batch):
    """Logits of -inf (a masked vocabulary: the first 40% and a band in the middle) in every row:
    whole chunks of some lanes hold no finite entry, and the masked tokens must never be drawn."""
    blocks = blocks_for(151936, temp, batch)
    w = wl.custom(seed=45, ctx=(0,) * len(blocks), block=blocks, vocab=151936)
    inp = wl.accept_inputs(w, temp)
    v = inp["target_logits"].shape[1]
    masked = np.zeros(v, dtype=bool)
    masked[: (4 * v) // 10] = True
    masked[v // 2: v // 2 + 5000] = True
    for key in ("target_logits", "draft_logits"):
        inp[key] = inp[key].copy()
        inp[key][:, masked] = -np.inf
    # redraw the drafted tokens from the masked draft rows (Gumbel-max at T>0, argmax at T=0)
    rng = np.random.default_rng([45, 99])
    d = inp["draft_logits"] / (temp if temp > 0 else 1.0)
    if temp > 0:
        d = d + rng.gumbel(size=d.shape).astype(np.float32)
    inp["draft_tokens"] = np.argmax(d, axis=1).astype(np.int32)
    compare_accept(inp, temp)
    _, out, _, _ = run_accept(inp, temp)
    emitted = out[out >= 0]
    assert not masked[emitted].any()


@pytest.mark.parametrize("batch", [False, True])
@pytest.mark.parametrize("temp", [1.0, 0.0])
def test_fully_masked_rows(temp, batch):
    """Some drafter rows and some target rows with every entry -inf.  Greedy: the argmax of a masked
    target row is index 0.  T > 0: a masked drafter row has q = 0, so its token is accepted when p > 0
    and the residual is p itself; no NaN reaches a decision."""
    blocks = blocks_for(3000, temp, batch)
    w = wl.custom(seed=46, ctx=(0,) * len(blocks), block=blocks, vocab=3000)
    inp = wl.accept_inputs(w, temp)
    inp["target_logits"] = inp["target_logits"].copy()
    inp["draft_logits"] = inp["draft_logits"].copy()
    cu = inp["cu_draft"]
    # per sequence with drafts: mask the drafter's first row; every third sequence (the one-row block
    # among them) also masks its target bonus row (greedy only: at T > 0 a masked target row has no
    # distribution to draw from)
    for s in range(len(blocks)):
        if cu[s + 1] > cu[s]:
            inp["draft_logits"][cu[s]] = -np.inf
        if temp == 0.0 and s % 3 == 1:
            inp["target_logits"][cu[s + 1] + s] = -np.inf
    compare_accept(inp, temp)
    n_acc, out, ap, status = run_accept(inp, temp)
    assert status == 0
    assert np.all(np.isfinite(ap))
    if temp == 0.0:
        assert out[cu[2] + 1] == 0  # sequence 1: one row, masked
