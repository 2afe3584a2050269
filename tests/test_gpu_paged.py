"""GPU parity of block attention over a paged KV cache, and of appending a block to the cache.

The oracle is the plain attention of oracle/ on the contiguous K/V rows the pages hold: paging
changes where rows live, not what the operation computes.  Same bars as the contiguous path.
"""
import numpy as np
import pytest
import torch

import paper_2606_31315_gb300 as bp
from paper_2606_31315_gb300 import workloads as wl

from _gpu import ATTN_TOL, LSE_TOL, attention_errors, attention_ws, dev, forced_split, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    bp.build()
    bp.load()


def _ragged():
    # contexts that end inside a page, a block longer than a 16-row page, one short sequence
    w = wl.custom(seed=11, ctx=(100, 700, 33, 1500), block=(8, 16, 5, 12), num_q_heads=32, num_kv_heads=8,
                  head_dim=128, dtype="bf16")
    return wl.attention_inputs(w)


def _run_paged(a, pk, mask, split="auto"):
    q = to_dev(a["q"], "bf16")
    kc, vc = to_dev(pk["k_cache"], "bf16"), to_dev(pk["v_cache"], "bf16")
    cu_q, cu_kv, bt = to_dev(a["cu_q"]), to_dev(a["cu_kv"]), to_dev(pk["block_table"])
    lse = torch.empty(q.shape[0], q.shape[1], dtype=torch.float32, device=dev())
    ws = attention_ws(a, split)
    with forced_split(split):
        o, _ = bp.block_attention_paged(q, kc, vc, cu_q, cu_kv, bt, pk["page_size"], int(a["cu_kv"][-1]),
                                        a["max_q_len"], a["max_kv_len"], mask=mask, lse=lse, ws=ws)
    assert bp.get_status(ws) == 0
    return o.float().cpu().numpy(), lse.cpu().numpy()


@pytest.mark.parametrize("page_size", [16, 64, 128, 256])
@pytest.mark.parametrize("mask", [bp.MASK_CAUSAL, bp.MASK_BIDIR])
@pytest.mark.parametrize("split", ["flat", "cluster"])
def test_paged_ragged_batch(page_size, mask, split):
    a = _ragged()
    pk = wl.paged_kv(a["k"], a["v"], a["cu_kv"], page_size, seed=page_size)
    o, lse = _run_paged(a, pk, mask, split)
    err, lerr = attention_errors(o, lse, a, mask, range(len(a["cu_q"]) - 1))
    assert err <= ATTN_TOL and lerr <= LSE_TOL, (err, lerr)


def test_paged_qwen3_4b_page64():
    a = wl.attention_inputs(wl.get("qwen3_4b"))
    pk = wl.paged_kv(a["k"], a["v"], a["cu_kv"], 64, seed=3)
    o, lse = _run_paged(a, pk, bp.MASK_CAUSAL)
    err, lerr = attention_errors(o, lse, a, bp.MASK_CAUSAL, [0])
    assert err <= ATTN_TOL and lerr <= LSE_TOL, (err, lerr)


@pytest.mark.parametrize("page_size", [16, 128])
def test_append_block_then_attend(page_size):
    # the cache holds only each sequence's context; bp_kv_append writes the block's K/V rows
    a = _ragged()
    cu_q, cu_kv = a["cu_q"], a["cu_kv"]
    blocks = np.diff(cu_q)
    ctx = np.diff(cu_kv) - blocks
    pk = wl.paged_kv(a["k"], a["v"], cu_kv, page_size, seed=5, rows_per_seq=ctx)
    rows = np.concatenate([np.arange(cu_kv[s] + ctx[s], cu_kv[s + 1]) for s in range(len(blocks))])
    kc, vc = to_dev(pk["k_cache"], "bf16"), to_dev(pk["v_cache"], "bf16")
    bt = to_dev(pk["block_table"])
    bp.kv_append(kc, vc, to_dev(a["k"][rows], "bf16"), to_dev(a["v"][rows], "bf16"), to_dev(cu_q), to_dev(cu_kv), bt,
                 page_size)
    torch.cuda.synchronize()
    # the pool now holds exactly the contiguous rows: attention over it matches the oracle
    pk["k_cache"], pk["v_cache"] = kc.view(torch.int16).cpu().numpy().view(np.uint16), \
        vc.view(torch.int16).cpu().numpy().view(np.uint16)
    full = wl.paged_kv(a["k"], a["v"], cu_kv, page_size, seed=5)
    np.testing.assert_array_equal(pk["k_cache"], full["k_cache"])
    np.testing.assert_array_equal(pk["v_cache"], full["v_cache"])
    o, lse = _run_paged(a, pk, bp.MASK_CAUSAL)
    err, lerr = attention_errors(o, lse, a, bp.MASK_CAUSAL, range(len(blocks)))
    assert err <= ATTN_TOL and lerr <= LSE_TOL, (err, lerr)
