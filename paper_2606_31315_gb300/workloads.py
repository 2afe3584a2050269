"""Seeded synthetic workloads for the block-verify hot path.

This module only draws random inputs of the right shapes and distributions; it holds
none of the method's arithmetic (no softmax, no acceptance test, no attention).  Both
the CUDA path and the CPU oracle are fed from it.

The five workloads stand in for the paper's evaluation data (GSM8K ... MT-Bench,
Section 3.1), which needs trained Qwen3 / DFlash models; they reproduce the shapes of
those models instead:

  tiny           1 seq, context 256, B=8, 4/2 heads, D=64, fp32, vocab 1024,
                 policy hidden 256 over 9 candidates
  qwen3_4b       1 seq, context 2048, B=16, 32/8 heads, D=128, bf16, vocab 151936
  ragged         32 seqs, B_s in {8..24} (60% on 14-18), context U[512, 8192],
                 Qwen3-4B heads, bf16, vocab 151936, policy N=32 over 2560-d states
  drafter_bidir  16 seqs, context 4096, B=16 mask-token queries, bidirectional
  long_context   8 seqs, context 32768, B=16, 32/8 heads, D=128, bf16, vocab 151936

Block of B query positions = the anchor token plus gamma = B - 1 drafted tokens; the
verify pass yields B target rows.  Draft tokens at T > 0 are drawn from the draft
distribution with the Gumbel-max trick (a sampler of the drafter, not of the
acceptance rule); at T = 0 they are the draft rows' argmax.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

CANDIDATES = np.arange(8, 25, 2, dtype=np.int32)  # {8, 10, ..., 24}


@dataclass(frozen=True)
class Workload:
    name: str
    seed: int
    num_seqs: int
    ctx: tuple  # per-sequence context length L_s (or a single value, repeated)
    block: tuple  # per-sequence block size B_s
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    dtype: str  # "f32" or "bf16"
    vocab: int
    logit_std: float
    temperatures: tuple
    mask: str = "causal"
    has_accept: bool = True
    policy: dict = field(default_factory=dict)


def _rng(seed: int, stream: int) -> np.random.Generator:
    return np.random.default_rng([seed, stream])


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bfloat16 (nearest, ties to even); returns the uint16 bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = u + 0x7FFF + ((u >> 16) & 1)
    return (u >> 16).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def _ragged_blocks(seed: int, n: int) -> tuple:
    sizes = np.array([8, 10, 12, 14, 16, 18, 20, 24])
    probs = np.array([0.08, 0.08, 0.08, 0.2, 0.2, 0.2, 0.08, 0.08])
    return tuple(int(b) for b in _rng(seed, 90).choice(sizes, size=n, p=probs))


def _ragged_ctx(seed: int, n: int) -> tuple:
    return tuple(int(c) for c in _rng(seed, 91).integers(512, 8192, size=n, endpoint=True))


def get(name: str) -> Workload:
    """The named workload (shapes and seeds fixed)."""
    if name == "tiny":
        return Workload("tiny", 0, 1, (256,), (8,), 4, 2, 64, "f32", 1024, 2.0, (1.0,),
                        policy=dict(num_reqs=1, d_in=1024, hidden=256, wdtype="f32", feat_std=2.0))
    if name == "qwen3_4b":
        return Workload("qwen3_4b", 2, 1, (2048,), (16,), 32, 8, 128, "bf16", 151936, 3.0, (1.0, 0.0))
    if name == "ragged":
        return Workload("ragged", 3, 32, _ragged_ctx(3, 32), _ragged_blocks(3, 32), 32, 8, 128, "bf16",
                        151936, 3.0, (1.0,),
                        policy=dict(num_reqs=32, d_in=2560, hidden=2048, wdtype="bf16", feat_std=1.0))
    if name == "drafter_bidir":
        return Workload("drafter_bidir", 4, 16, (4096,) * 16, (16,) * 16, 32, 8, 128, "bf16", 151936, 3.0,
                        (), mask="bidir", has_accept=False)
    if name == "long_context":
        return Workload("long_context", 5, 8, (32768,) * 8, (16,) * 8, 32, 8, 128, "bf16", 151936, 3.0,
                        (0.0, 1.0))
    raise KeyError(name)


NAMES = ("tiny", "qwen3_4b", "ragged", "drafter_bidir", "long_context")


def custom(name="custom", seed=0, ctx=(64,), block=(8,), num_q_heads=4, num_kv_heads=2, head_dim=128,
           dtype="bf16", vocab=1000, logit_std=3.0, temperatures=(1.0,), mask="causal", policy=None) -> Workload:
    """A workload of arbitrary shape (used for small parity cases and edge cases)."""
    ctx = tuple(int(c) for c in ctx)
    block = tuple(int(b) for b in block)
    assert len(ctx) == len(block)
    return Workload(name, seed, len(ctx), ctx, block, num_q_heads, num_kv_heads, head_dim, dtype, vocab,
                    logit_std, tuple(temperatures), mask=mask, policy=policy or {})


def offsets(lengths) -> np.ndarray:
    out = np.zeros(len(lengths) + 1, dtype=np.int32)
    out[1:] = np.cumsum(np.asarray(lengths, dtype=np.int64))
    return out


def attention_inputs(w: Workload) -> dict:
    """Q [sum B_s, Hq, D], K/V [sum (L_s + B_s), Hkv, D] ~ N(0,1) and the ragged offsets.

    For bf16 workloads the arrays are uint16 bf16 bits; for f32 they are float32.
    """
    blocks = np.asarray(w.block, dtype=np.int64)
    kv_lens = np.asarray(w.ctx, dtype=np.int64) + blocks
    cu_q = offsets(blocks)
    cu_kv = offsets(kv_lens)
    tq, tkv = int(cu_q[-1]), int(cu_kv[-1])
    out = dict(cu_q=cu_q, cu_kv=cu_kv, num_q_heads=w.num_q_heads, num_kv_heads=w.num_kv_heads,
               head_dim=w.head_dim, dtype=w.dtype, mask=w.mask, max_q_len=int(blocks.max(initial=0)),
               max_kv_len=int(kv_lens.max(initial=0)))
    shapes = dict(q=(tq, w.num_q_heads, w.head_dim), k=(tkv, w.num_kv_heads, w.head_dim),
                  v=(tkv, w.num_kv_heads, w.head_dim))
    for i, key in enumerate(("q", "k", "v")):
        x = _rng(w.seed, 10 + i).standard_normal(shapes[key], dtype=np.float32)
        out[key] = f32_to_bf16_bits(x) if w.dtype == "bf16" else x
    return out


def paged_kv(k: np.ndarray, v: np.ndarray, cu_kv, page_size: int, seed: int = 0, spare_pages: int = 3,
             rows_per_seq=None) -> dict:
    """Scatters contiguous K/V rows [total_kv, Hkv, D] into a pool of pages of page_size rows, the
    pages of every sequence in shuffled order, as a serving engine's cache would hold them.

    Rows of the pool no sequence owns are filled with other seeded values (finite), so a wrong
    page lookup changes the result.  rows_per_seq (default: all of each sequence's rows) limits
    how many leading rows of each sequence are copied in; the block table still covers all of
    cu_kv's rows, so the rest can be appended later.  Returns the pools, the block table
    [S, pages_per_seq] and the page count."""
    cu_kv = np.asarray(cu_kv, dtype=np.int64)
    s_count = len(cu_kv) - 1
    lens = np.diff(cu_kv)
    pages = [int((l + page_size - 1) // page_size) for l in lens]
    pps = max(1, max(pages) if s_count else 1)
    n_pages = int(sum(pages)) + spare_pages
    rng = _rng(seed, 40)
    perm = rng.permutation(n_pages)
    hkv, d = k.shape[1], k.shape[2]
    fill = rng.standard_normal((n_pages * page_size, hkv, d), dtype=np.float32)
    if k.dtype == np.uint16:  # bf16 bits
        fill = f32_to_bf16_bits(fill)
    else:
        fill = fill.astype(k.dtype)
    kp, vp = fill.copy(), fill[::-1].copy()
    table = np.full((s_count, pps), perm[-1], dtype=np.int32)
    idx = 0
    for sq in range(s_count):
        keep = int(lens[sq]) if rows_per_seq is None else int(rows_per_seq[sq])
        for pi in range(pages[sq]):
            page = int(perm[idx])
            idx += 1
            table[sq, pi] = page
            lo = pi * page_size
            hi = min(keep, lo + page_size)
            if hi > lo:
                src = slice(int(cu_kv[sq]) + lo, int(cu_kv[sq]) + hi)
                kp[page * page_size:page * page_size + hi - lo] = k[src]
                vp[page * page_size:page * page_size + hi - lo] = v[src]
    return dict(k_cache=kp, v_cache=vp, block_table=table, num_pages=n_pages, page_size=page_size)


def accept_inputs(w: Workload, temperature: float, planted_match: float = 0.0) -> dict:
    """Target / draft logits, draft tokens and uniforms for one acceptance step.

    target rows ~ N(0, logit_std^2) [sum (gamma_s + 1), V]; draft rows = matching target
    row + N(0, 1) [sum gamma_s, V]; gamma_s = B_s - 1.  With planted_match > 0 each draft
    row is, with that probability, an exact copy of its target row (full agreement).
    """
    gammas = np.asarray(w.block, dtype=np.int64) - 1
    cu_draft = offsets(gammas)
    s = w.num_seqs
    td = int(cu_draft[-1])
    V = w.vocab
    target = _rng(w.seed, 20).standard_normal((td + s, V), dtype=np.float32) * np.float32(w.logit_std)
    noise = _rng(w.seed, 21).standard_normal((td, V), dtype=np.float32)
    # target row index of drafted position i of sequence s is cu_draft[s] + s + i
    seq_of_draft = np.repeat(np.arange(s), gammas)
    trow = np.arange(td) + seq_of_draft
    draft = target[trow] + noise
    if planted_match > 0.0:
        copy = _rng(w.seed, 22).random(td) < planted_match
        draft[copy] = target[trow[copy]]
    if temperature > 0.0:
        g = _rng(w.seed, 23).gumbel(size=(td, V)).astype(np.float32)
        tokens = np.argmax(draft / np.float32(temperature) + g, axis=1).astype(np.int32)
    else:
        tokens = np.argmax(draft, axis=1).astype(np.int32)
    u_accept = _rng(w.seed, 24).random(td, dtype=np.float32)
    u_sample = _rng(w.seed, 25).random(s, dtype=np.float32)
    return dict(target_logits=target, draft_logits=draft, draft_tokens=tokens, cu_draft=cu_draft,
                u_accept=u_accept, u_sample=u_sample, vocab=V, temperature=float(temperature))


def policy_inputs(w: Workload) -> dict:
    """Pooled-feature matrix (4 prefill rows per request, the last one pooled) and MLP weights."""
    p = w.policy
    n, d_in, hidden = p["num_reqs"], p["d_in"], p["hidden"]
    c = len(CANDIDATES)
    rows_per_req = 4
    feats = _rng(w.seed, 30).standard_normal((n * rows_per_req, d_in), dtype=np.float32) * np.float32(p["feat_std"])
    row_index = (np.arange(n, dtype=np.int32) * rows_per_req + rows_per_req - 1).astype(np.int32)
    w1 = _rng(w.seed, 31).standard_normal((hidden, d_in), dtype=np.float32) * np.float32(1.0 / np.sqrt(d_in))
    b1 = _rng(w.seed, 32).standard_normal(hidden, dtype=np.float32) * np.float32(0.1)
    w2 = _rng(w.seed, 33).standard_normal((c, hidden), dtype=np.float32) * np.float32(1.0 / np.sqrt(hidden))
    b2 = _rng(w.seed, 34).standard_normal(c, dtype=np.float32) * np.float32(0.1)
    out = dict(row_index=row_index, b1=b1, b2=b2, candidates=CANDIDATES.copy(), wdtype=p["wdtype"])
    if p["wdtype"] == "bf16":
        out.update(feats=f32_to_bf16_bits(feats), w1=f32_to_bf16_bits(w1), w2=f32_to_bf16_bits(w2))
    else:
        out.update(feats=feats, w1=w1, w2=w2)
    return out


# hidden size of the final states the LM head projects (Qwen3-4B: 2560)
LM_HIDDEN = {"tiny": 128, "qwen3_4b": 2560, "ragged": 2560, "long_context": 2560}


def lm_head_weight(vocab: int, hidden: int, logit_std: float, seed: int) -> np.ndarray:
    """LM-head weight [V, H] ~ N(0, logit_std^2 / H) as bf16 bits (so unit-variance states get
    logits ~ N(0, logit_std^2)); drawn and rounded in chunks of rows to bound host memory."""
    rng = _rng(seed, 50)
    out = np.empty((vocab, hidden), dtype=np.uint16)
    scale = np.float32(logit_std / np.sqrt(hidden))
    step = max(1, (1 << 24) // hidden)
    for r0 in range(0, vocab, step):
        r1 = min(vocab, r0 + step)
        out[r0:r1] = f32_to_bf16_bits(rng.standard_normal((r1 - r0, hidden), dtype=np.float32) * scale)
    return out


def lm_head_inputs(w: Workload, temperature: float, hidden: int | None = None, push_prob: float = 0.85,
                   boost: float = 18.0, weight: np.ndarray | None = None, target_peak: float | None = None) -> dict:
    """LM-head weight, the final hidden states the verify epilogue projects, draft tokens, uniforms.

    W [V, H] from lm_head_weight.  Target states [sum (gamma_s + 1), H] ~ N(0, 1).  Draft token x_i
    is uniform over V.  The drafter's state of position i is its target row's state plus
    N(0, 1 / logit_std^2) noise (its logits are the target's plus unit-variance noise) plus
    boost * w_x / |w_x|^2, which raises the drafter's logit of x_i by `boost`; with probability
    push_prob the target row's state gets the same push (the target agrees with the draft),
    otherwise none.  With target_peak, every target row not pushed toward its draft (the rows of
    rejected drafts and each sequence's last row) is pushed the same way toward a random token of
    its own by target_peak, giving it a dominant token as a confident model's rows have.  States are
    rounded to bf16 last.  At T = 0 the drafter's states are not returned (greedy acceptance reads
    the target rows only).
    """
    gammas = np.asarray(w.block, dtype=np.int64) - 1
    cu_draft = offsets(gammas)
    s = w.num_seqs
    td = int(cu_draft[-1])
    V = w.vocab
    H = hidden or LM_HIDDEN.get(w.name, 256)
    W = weight if weight is not None else lm_head_weight(V, H, w.logit_std, w.seed)
    base = _rng(w.seed, 51).standard_normal((td + s, H)).astype(np.float64)
    noise = _rng(w.seed, 52).standard_normal((td, H)) / w.logit_std
    tokens = _rng(w.seed, 53).integers(0, V, size=td).astype(np.int32)
    push = _rng(w.seed, 54).random(td) < push_prob
    seq_of_draft = np.repeat(np.arange(s), gammas)
    trow = np.arange(td) + seq_of_draft  # target row of drafted position i
    wx = bf16_bits_to_f32(W[tokens]).astype(np.float64) if td else np.zeros((0, H))
    dirs = wx / np.maximum((wx * wx).sum(axis=1, keepdims=True), 1e-30) * boost
    h_draft = base[trow] + noise + dirs
    h_target = base.copy()
    h_target[trow[push]] += dirs[push]
    if target_peak is not None:
        free = np.ones(td + s, dtype=bool)
        free[trow[push]] = False
        fav = _rng(w.seed, 57).integers(0, V, size=td + s)
        wf = bf16_bits_to_f32(W[fav[free]]).astype(np.float64)
        h_target[free] += wf / np.maximum((wf * wf).sum(axis=1, keepdims=True), 1e-30) * target_peak
    out = dict(w=W, hidden=H, h_target=f32_to_bf16_bits(h_target.astype(np.float32)), draft_tokens=tokens,
               cu_draft=cu_draft, vocab=V, temperature=float(temperature),
               u_accept=_rng(w.seed, 55).random(td, dtype=np.float32),
               u_sample=_rng(w.seed, 56).random(s, dtype=np.float32))
    out["h_draft"] = f32_to_bf16_bits(h_draft.astype(np.float32)) if temperature > 0.0 else None
    return out


def tau_inputs(num_reqs: int, jmax: int = 24, seed: int = 60, train_block: int = 16, alpha: float = 0.001) -> dict:
    """Per-request predictabilities for Appendix A's acceptance-length model and a predicted block size.

    gamma_x ~ Beta(12, 2) per request (mean 0.86: tau(16) near the paper's 5.92 at B = 16); per
    position gamma_j = clip(gamma_x + N(0, 0.03^2), 0.05, 0.999), [num_reqs, jmax] fp32.  The
    predicted size is the candidate nearest to train_block + N(0, 1.5^2) (a predictor that
    concentrates near the training size).  alpha is the retention constant of the model.
    """
    rng = _rng(seed, 61)
    gx = rng.beta(12.0, 2.0, size=num_reqs).astype(np.float32)
    noise = _rng(seed, 62).standard_normal((num_reqs, jmax), dtype=np.float32) * np.float32(0.03)
    gamma = np.clip(gx[:, None] + noise, np.float32(0.05), np.float32(0.999)).astype(np.float32)
    want = train_block + _rng(seed, 63).standard_normal(num_reqs) * 1.5
    idx = np.abs(want[:, None] - CANDIDATES[None, :]).argmin(axis=1)
    return dict(gamma=gamma, candidates=CANDIDATES.copy(), predicted=CANDIDATES[idx].astype(np.int32),
                train_block=int(train_block), alpha=float(alpha))


def as_f64(x: np.ndarray, dtype: str) -> np.ndarray:
    """The exact fp64 values of an f32 array or of bf16 bits."""
    if dtype == "bf16":
        return bf16_bits_to_f32(x).astype(np.float64)
    return np.asarray(x, dtype=np.float32).astype(np.float64)
