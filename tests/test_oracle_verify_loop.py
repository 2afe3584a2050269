"""Pins of the oracle's commit of a verify step (the decoding loop of Section 2.1 / Figure 1): over
several steps the tokens whose K/V rows stay in a sequence's cache are exactly its text so far minus
the last token, and that last token is the next anchor -- tracked here by building the text from the
accepted drafts and emitted tokens, not from the commit rule."""
import numpy as np
import pytest

import oracle
from paper_2606_31315_gb300 import workloads as wl


def test_cache_holds_the_text_but_its_last_token():
    rng = np.random.default_rng(0)
    blocks = (8, 5, 16, 1)
    S = len(blocks)
    gammas = np.array(blocks) - 1
    cu_draft = wl.offsets(gammas)
    td = int(cu_draft[-1])
    V = 50
    ctx = np.array([20, 3, 64, 9], dtype=np.int32)
    text = [list(rng.integers(0, V, size=c + 1)) for c in ctx]  # prompt + the first anchor
    cache = [t[:-1] for t in text]  # rows in the cache: everything but the anchor
    anchor = np.array([t[-1] for t in text], dtype=np.int32)
    for step in range(6):
        # the block of each sequence: its anchor and gamma drafts; their rows are appended
        drafts = rng.integers(0, V, size=td).astype(np.int32)
        for s in range(S):
            cache[s] = cache[s] + [int(anchor[s])] + list(drafts[cu_draft[s]:cu_draft[s + 1]])
        # greedy acceptance on logits that agree with the drafts now and then
        target = rng.normal(size=(td + S, V))
        for i in range(td):
            if rng.random() < 0.7:
                seq = np.searchsorted(cu_draft, i, side="right") - 1
                target[i + seq, drafts[i]] = 10.0
        acc = oracle.spec_accept(target, None, drafts, cu_draft, 0.0)
        res = oracle.verify_commit(ctx, acc["n_accepted"], acc["out_tokens"], cu_draft, capacity=10_000)
        for s in range(S):
            k = int(acc["n_accepted"][s])
            emitted = int(acc["out_tokens"][cu_draft[s] + s + k])
            text[s] = text[s] + list(drafts[cu_draft[s]:cu_draft[s] + k]) + [emitted]
            cache[s] = cache[s][:res["ctx"][s]]  # rows past the new length are discarded
            assert cache[s] == text[s][:-1], (step, s)
            assert res["anchor"][s] == text[s][-1]
        np.testing.assert_array_equal(np.diff(res["cu_kv"]), res["ctx"] + np.array(blocks))
        ctx, anchor = res["ctx"], res["anchor"]


def test_refusals_change_nothing():
    cu = np.array([0, 3, 4], dtype=np.int32)
    out = np.array([7, 8, 9, -1, 3, -1], dtype=np.int32)
    with pytest.raises(ValueError):
        oracle.verify_commit([10, 5], [4, 0], out, cu, 100)  # more accepted than drafted
    with pytest.raises(ValueError):
        oracle.verify_commit([10, 5], [3, 1], out, cu, 17)  # 10 + 4 + 4 rows > 17
