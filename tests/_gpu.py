"""Helpers for the GPU parity tests: move seeded workloads to the device, run the CUDA path
through the C ABI, run the oracle on the same inputs (whole or sampled) and compare."""
from __future__ import annotations

import contextlib
import os

import numpy as np
import torch

import oracle
import paper_2606_31315_gb300 as bp
from paper_2606_31315_gb300 import workloads as wl

ATTN_TOL = 2e-2      # max |O - O_ref| / max |O_ref| per (sequence, query head) slice
LSE_TOL = 2e-3       # absolute, natural-log units
PROB_TOL = 1e-5      # accept_prob absolute
FLAG = 1e-5          # near-tie flag for ratio test and inverse-CDF draws


def dev():
    return torch.device("cuda:0")


def to_dev(x: np.ndarray, dtype: str | None = None) -> torch.Tensor:
    if dtype == "bf16":
        return torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).to(dev()).view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(x)).to(dev())


def attention_ws(a: dict, split: str = "auto"):
    """A workspace for the attention of workload a: the size the library asks for, or (split "cluster")
    the 256-byte header alone, which keeps the cluster split of the bf16 path."""
    if split == "cluster":
        return bp.workspace(256, dev())
    return bp.workspace(bp.block_attention_workspace_size(len(a["cu_q"]) - 1, a["max_q_len"], a["num_q_heads"],
                                                          a["num_kv_heads"], a["head_dim"]), dev())


@contextlib.contextmanager
def forced_split(split: str):
    """The library's choice between the flat and the cluster split of the keys ("auto"), or one of them
    forced through BP_ATTENTION_SPLIT, which the library reads at every call ("cluster3": the cluster
    split in clusters of 3, so that short contexts too take the distributed-shared-memory merge)."""
    old = os.environ.get("BP_ATTENTION_SPLIT")
    if split in ("flat", "cluster"):
        os.environ["BP_ATTENTION_SPLIT"] = split
    elif split == "cluster3":
        os.environ["BP_ATTENTION_SPLIT"] = "cluster:3"
    else:
        os.environ.pop("BP_ATTENTION_SPLIT", None)
    try:
        yield
    finally:
        if old is None:
            os.environ.pop("BP_ATTENTION_SPLIT", None)
        else:
            os.environ["BP_ATTENTION_SPLIT"] = old


def run_attention(a: dict, mask: int, split: str = "auto"):
    """CUDA path on the whole workload; returns (o fp32 numpy, lse numpy).  split: "auto" (the library
    chooses), "flat", "cluster" or "cluster3" (forced)."""
    q, k, v = to_dev(a["q"], a["dtype"]), to_dev(a["k"], a["dtype"]), to_dev(a["v"], a["dtype"])
    cu_q, cu_kv = to_dev(a["cu_q"]), to_dev(a["cu_kv"])
    lse = torch.empty(q.shape[0], q.shape[1], dtype=torch.float32, device=dev())
    ws = attention_ws(a, split)
    with forced_split(split):
        o, _ = bp.block_attention(q, k, v, cu_q, cu_kv, a["max_q_len"], a["max_kv_len"], mask=mask, lse=lse, ws=ws)
    assert bp.get_status(ws) == 0
    return o.float().cpu().numpy(), lse.cpu().numpy()


def oracle_attention_slice(a: dict, s: int, kv_head: int | None, mask: int):
    """Oracle on sequence s (all heads, or the query heads of one KV head); returns the
    (o, lse) rows of that sequence and the q-head indices covered."""
    cq, ck = a["cu_q"], a["cu_kv"]
    hq, hkv = a["num_q_heads"], a["num_kv_heads"]
    g = hq // hkv
    heads = np.arange(hq) if kv_head is None else np.arange(kv_head * g, (kv_head + 1) * g)
    kvh = np.arange(hkv) if kv_head is None else np.array([kv_head])
    q = wl.as_f64(a["q"][cq[s]:cq[s + 1]][:, heads], a["dtype"])
    k = wl.as_f64(a["k"][ck[s]:ck[s + 1]][:, kvh], a["dtype"])
    v = wl.as_f64(a["v"][ck[s]:ck[s + 1]][:, kvh], a["dtype"])
    o, lse = oracle.block_attention(q, k, v, [0, q.shape[0]], [0, k.shape[0]], len(kvh), mask)
    return o, lse, heads


def attention_errors(o_gpu, lse_gpu, a: dict, mask: int, seqs, kv_head: int | None = None):
    """Worst per-(sequence, head) relative error and worst lse error over the sampled sequences."""
    worst, worst_lse = 0.0, 0.0
    for s in seqs:
        cq = a["cu_q"]
        if cq[s + 1] == cq[s]:
            continue
        o_ref, lse_ref, heads = oracle_attention_slice(a, s, kv_head, mask)
        got = o_gpu[cq[s]:cq[s + 1]][:, heads]
        for hi in range(len(heads)):
            denom = np.abs(o_ref[:, hi]).max()
            worst = max(worst, np.abs(got[:, hi] - o_ref[:, hi]).max() / max(denom, 1e-30))
        worst_lse = max(worst_lse, np.abs(lse_gpu[cq[s]:cq[s + 1]][:, heads] - lse_ref).max())
    return worst, worst_lse


# The library's choice between its two acceptance arrangements, mirrored so that tests can take both
# sides: the throughput kernels from this many logits read on (target rows x vocab at T = 0, target and
# drafter rows x vocab at T > 0), the per-row cluster kernel below it.
BATCH_LOGITS_T0, BATCH_LOGITS_T1 = 2_500_000, 6_500_000


def accept_uses_batch(blocks, vocab: int, temperature: float) -> bool:
    s, td = len(blocks), int(np.sum(blocks)) - len(blocks)
    rows = td + s if temperature == 0 else 2 * td + s
    return rows * vocab >= (BATCH_LOGITS_T0 if temperature == 0 else BATCH_LOGITS_T1)


SMALL_BLOCK_SETS = ((16, 1, 3, 9, 8), (16, 9, 1), (16, 9), (9, 1, 3), (4, 1))
LARGE_BLOCKS = (16, 1, 3, 9, 24, 16, 5, 2, 16)


def blocks_for(vocab: int, temperature: float, batch: bool) -> tuple:
    """Ragged blocks (1 to 24 positions) whose acceptance at this vocabulary and temperature runs on the
    throughput kernels (batch) or on the cluster kernel."""
    if batch:
        n = 1
        while not accept_uses_batch(LARGE_BLOCKS * n, vocab, temperature):
            n += 1
        return LARGE_BLOCKS * n
    for b in SMALL_BLOCK_SETS:
        if not accept_uses_batch(b, vocab, temperature):
            return b
    raise ValueError("no small block set for this vocabulary")


def run_accept(inp: dict, temperature: float, ws=None):
    g = {key: to_dev(inp[key]) for key in ("target_logits", "draft_tokens", "cu_draft", "u_accept", "u_sample")}
    draft = to_dev(inp["draft_logits"]) if temperature > 0 else None
    s = len(inp["cu_draft"]) - 1
    if ws is None:
        ws = bp.workspace(bp.spec_accept_workspace_size(s, int(inp["cu_draft"][-1]), inp["target_logits"].shape[1]),
                          dev())
    n_acc, out, ap = bp.spec_accept(g["target_logits"], draft, g["draft_tokens"], g["cu_draft"], temperature,
                                    g["u_accept"], g["u_sample"], ws=ws)
    status = bp.get_status(ws)
    return n_acc.cpu().numpy(), out.cpu().numpy(), ap.cpu().numpy(), status


def run_oracle_accept(inp: dict, temperature: float):
    return oracle.spec_accept(inp["target_logits"], inp["draft_logits"] if temperature > 0 else None,
                              inp["draft_tokens"], inp["cu_draft"], temperature, inp["u_accept"], inp["u_sample"])


def _near_tie_tokens(inp: dict, s: int, k: int, temperature: float) -> np.ndarray:
    """Tokens whose fp64 inverse-CDF interval lies within FLAG of the draw's threshold (sequence s,
    emitting at slot k).  Used only for sequences the oracle flags as near-ties."""
    from scipy import special

    cu = inp["cu_draft"]
    gamma = cu[s + 1] - cu[s]
    p = special.softmax(inp["target_logits"][cu[s] + s + k].astype(np.float64) / temperature)
    w = p
    if k < gamma:
        q = special.softmax(inp["draft_logits"][cu[s] + k].astype(np.float64) / temperature)
        r = np.maximum(p - q, 0.0)
        if r.sum() > 0:
            w = r
    c = np.cumsum(w)
    thr = float(inp["u_sample"][s]) * c[-1]
    prev = np.concatenate([[0.0], c[:-1]])
    return np.nonzero((w > 0) & (prev - FLAG <= thr) & (thr < c + FLAG))[0]


def compare_accept(inp: dict, temperature: float, gpu=None, ref=None):
    """Asserts parity.  Unflagged sequences: n_accepted and out_tokens bit-exact.  Flagged sequences
    (near-ties): the GPU's prefix must follow from its own accept_prob (which is within 1e-5 of
    the oracle's), the positions where it departs from the oracle must be near-ties, and its
    emitted token must lie in the fp64 near-tie set.  Returns (flagged, sequences)."""
    n_acc, out, ap, status = gpu if gpu is not None else run_accept(inp, temperature)
    ref = ref if ref is not None else run_oracle_accept(inp, temperature)
    assert status == 0, f"device error status {status}"
    cu = inp["cu_draft"]
    s = len(cu) - 1
    assert np.abs(ap - ref["accept_prob"]).max(initial=0.0) <= PROB_TOL, np.abs(ap - ref["accept_prob"]).max()
    flagged = (ref["ratio_margin"] < FLAG) | (ref["cdf_margin"] < FLAG)
    if temperature == 0:
        assert not flagged.any()
    for i in range(s):
        lo, hi = cu[i] + i, cu[i + 1] + i + 1
        gamma = cu[i + 1] - cu[i]
        k = int(n_acc[i])
        if temperature > 0:
            # the GPU's prefix is the ratio test applied to its own a_i
            ua = inp["u_accept"][cu[i]:cu[i + 1]]
            rej = np.nonzero(~(ua < ap[cu[i]:cu[i + 1]]))[0]
            assert k == (rej[0] if len(rej) else gamma), (i, k, rej)
        if not flagged[i]:
            assert k == ref["n_accepted"][i], (i, k, ref["n_accepted"][i])
            np.testing.assert_array_equal(out[lo:hi], ref["out_tokens"][lo:hi], err_msg=f"sequence {i}")
            continue
        kr = int(ref["n_accepted"][i])
        if k != kr:  # a departure of the prefix is allowed only at a ratio-test near-tie
            j = min(k, kr)
            assert abs(float(inp["u_accept"][cu[i] + j]) - ref["accept_prob"][cu[i] + j]) < FLAG, (i, k, kr)
        np.testing.assert_array_equal(out[lo:lo + k], inp["draft_tokens"][cu[i]:cu[i] + k])
        assert np.all(out[lo + k + 1:hi] == -1)
        assert out[lo + k] in _near_tie_tokens(inp, i, k, temperature), (i, k, out[lo + k])
    return int(flagged.sum()), s
