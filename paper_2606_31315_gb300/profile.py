"""One kernel of the hot path on its own, for profilers: seeded synthetic inputs of the benchmark's
shapes on the device (nothing else allocated), a few warm-up calls, then N calls.

    python -m paper_2606_31315_gb300.profile CASE [--calls N] [--warmup W] [--split flat|cluster]

CASE is one of:
  verify_epilogue_t1  Qwen3-4B LM head (151936 x 2560 bf16) fused with the acceptance, 16 target and
                      15 drafter states, T = 1
  verify_epilogue_t0  the same at T = 0 (16 target states)
  verify_stream_c5_t1 the long-context batch through the same LM head: 8 sequences x 16 positions,
                      128 target and 120 drafter states (248 rows, streamed), T = 1
  verify_stream_c5_t0 the same at T = 0 (128 target states)
  accept_t1           acceptance over 16 x 151936 target and 15 x 151936 draft fp32 logits, T = 1
  accept_batch_t1     acceptance over a batch of 32 sequences of 16 target rows (512 x 151936 target
                      and 480 x 151936 draft fp32 logits), T = 1: the three throughput kernels
  accept_batch_t0     the same batch at T = 0 (target logits only)
  attention           causal verify attention, 1 sequence, 2048 + 16 keys, 32 / 8 heads, D = 128
  attention_c3        causal verify attention over the ragged batch: 32 sequences, blocks 8..24,
                      contexts 562..8118 (576 MB of K/V)
  attention_c5        causal verify attention over the long-context batch: 8 sequences of 32768 + 16
                      keys (1.07 GB of K/V)
  accept_c5_t1        acceptance of the long-context batch at T = 1: 8 x 16 target and 8 x 15 draft
                      rows over 151936 (150.7 MB): the three throughput kernels
  step_c5             one long-context verify step: attention_c5, then accept_c5_t1
  policy              policy head, 32 requests, 2560 -> 2048 -> 9 bf16 (W1 loaded at once per CTA)
  policy_d151936      policy head at the paper's input width, 32 requests, 151936 -> 2048 -> 9 bf16
                      (W1 622 MB streamed through the ring)
  tau                 Appendix A's acceptance-length model over 4M requests (24 positions, nine
                      candidate sizes, a predicted size each)
"""
from __future__ import annotations

import argparse
import itertools

import torch

from . import _binding as bp

V, H, CTX, B, HQ, HKV, D = 151936, 2560, 2048, 16, 32, 8, 128
SPLIT = {"split": "flat"}  # attention cases: a full-size workspace (flat split) or the 256-byte header (cluster split)


def _attn_ws(dev, num_seqs, max_q):
    if SPLIT["split"] == "cluster":
        return bp.workspace(256, dev)
    return bp.workspace(bp.block_attention_workspace_size(num_seqs, max_q, HQ, HKV, D), dev)


def _verify_epilogue(dev, gen, temperature):
    td = B - 1
    w = (torch.randn(V, H, device=dev, generator=gen) * (3.0 / H ** 0.5)).to(torch.bfloat16)
    h_t = torch.randn(td + 1, H, device=dev, generator=gen).to(torch.bfloat16)
    h_d = (h_t[:td].float() + torch.randn(td, H, device=dev, generator=gen) / 3).to(torch.bfloat16)
    tok = torch.randint(0, V, (td,), device=dev, generator=gen, dtype=torch.int32)
    cu = torch.tensor([0, td], dtype=torch.int32, device=dev)
    ua, us = torch.rand(td, device=dev, generator=gen), torch.rand(1, device=dev, generator=gen)
    ws = bp.workspace(bp.verify_epilogue_workspace_size(1, td, V), dev)
    return lambda: bp.verify_epilogue(w, h_t, h_d if temperature > 0 else None, tok, cu, temperature, ua, us,
                                      want_accept_prob=False, ws=ws)


def _verify_stream_c5(dev, gen, temperature):
    S, td = 8, 8 * (B - 1)
    w = (torch.randn(V, H, device=dev, generator=gen) * (3.0 / H ** 0.5)).to(torch.bfloat16)
    h_t = torch.randn(td + S, H, device=dev, generator=gen).to(torch.bfloat16)
    h_d = torch.randn(td, H, device=dev, generator=gen).to(torch.bfloat16)
    tok = torch.randint(0, V, (td,), device=dev, generator=gen, dtype=torch.int32)
    cu = torch.arange(0, td + 1, B - 1, dtype=torch.int32, device=dev)
    ua, us = torch.rand(td, device=dev, generator=gen), torch.rand(S, device=dev, generator=gen)
    ws = bp.workspace(bp.verify_epilogue_workspace_size(S, td, V), dev)
    return lambda: bp.verify_epilogue(w, h_t, h_d if temperature > 0 else None, tok, cu, temperature, ua, us,
                                      want_accept_prob=False, ws=ws)


def _accept(dev, gen):
    td = B - 1
    t = torch.randn(td + 1, V, device=dev, generator=gen) * 3
    d = t[:td] + torch.randn(td, V, device=dev, generator=gen)
    tok = torch.randint(0, V, (td,), device=dev, generator=gen, dtype=torch.int32)
    cu = torch.tensor([0, td], dtype=torch.int32, device=dev)
    ua, us = torch.rand(td, device=dev, generator=gen), torch.rand(1, device=dev, generator=gen)
    ws = bp.workspace(bp.spec_accept_workspace_size(1, td, V), dev)
    return lambda: bp.spec_accept(t, d, tok, cu, 1.0, ua, us, ws=ws)


def _accept_batch(dev, gen, temperature):
    s = 32
    td = s * (B - 1)
    t = torch.randn(td + s, V, device=dev, generator=gen) * 3
    d = torch.randn(td, V, device=dev, generator=gen) * 3 if temperature > 0 else None
    tok = torch.randint(0, V, (td,), device=dev, generator=gen, dtype=torch.int32)
    cu = torch.arange(0, td + 1, B - 1, dtype=torch.int32, device=dev)
    ua, us = torch.rand(td, device=dev, generator=gen), torch.rand(s, device=dev, generator=gen)
    ws = bp.workspace(bp.spec_accept_workspace_size(s, td, V), dev)
    return lambda: bp.spec_accept(t, d, tok, cu, temperature, ua, us, ws=ws)


def _attention(dev, gen):
    q = torch.randn(B, HQ, D, device=dev, generator=gen).to(torch.bfloat16)
    k = torch.randn(CTX + B, HKV, D, device=dev, generator=gen).to(torch.bfloat16)
    v = torch.randn(CTX + B, HKV, D, device=dev, generator=gen).to(torch.bfloat16)
    cu_q = torch.tensor([0, B], dtype=torch.int32, device=dev)
    cu_kv = torch.tensor([0, CTX + B], dtype=torch.int32, device=dev)
    ws = _attn_ws(dev, 1, B)
    return lambda: bp.block_attention(q, k, v, cu_q, cu_kv, B, CTX + B, mask=bp.MASK_CAUSAL, ws=ws)


def _batch_attention(dev, gen, ctx, block):
    """Causal verify attention over sequences of the given contexts and blocks (Qwen3 heads)."""
    kv = [c + b for c, b in zip(ctx, block)]
    q = torch.randn(sum(block), HQ, D, device=dev, generator=gen).to(torch.bfloat16)
    k = torch.randn(sum(kv), HKV, D, device=dev, generator=gen).to(torch.bfloat16)
    v = torch.randn(sum(kv), HKV, D, device=dev, generator=gen).to(torch.bfloat16)
    off = lambda xs: torch.tensor([0] + list(itertools.accumulate(xs)), dtype=torch.int32, device=dev)  # noqa
    cu_q, cu_kv = off(block), off(kv)
    ws = _attn_ws(dev, len(ctx), max(block))
    return lambda: bp.block_attention(q, k, v, cu_q, cu_kv, max(block), max(kv), mask=bp.MASK_CAUSAL, ws=ws)


def _accept_c5(dev, gen):
    s, td = 8, 8 * (B - 1)
    t = torch.randn(td + s, V, device=dev, generator=gen) * 3
    trow = torch.tensor([i + i // (B - 1) for i in range(td)], device=dev)
    d = t[trow] + torch.randn(td, V, device=dev, generator=gen)
    tok = torch.randint(0, V, (td,), device=dev, generator=gen, dtype=torch.int32)
    cu = torch.arange(0, td + 1, B - 1, dtype=torch.int32, device=dev)
    ua, us = torch.rand(td, device=dev, generator=gen), torch.rand(s, device=dev, generator=gen)
    ws = bp.workspace(bp.spec_accept_workspace_size(s, td, V), dev)
    return lambda: bp.spec_accept(t, d, tok, cu, 1.0, ua, us, want_accept_prob=False, ws=ws)


def _step_c5(dev, gen):
    attn = _batch_attention(dev, gen, [32768] * 8, [B] * 8)
    acc = _accept_c5(dev, gen)

    def step():
        attn()
        acc()
    return step


def _ragged_shapes():
    from . import workloads

    w = workloads.get("ragged")
    return list(w.ctx), list(w.block)


def _policy(dev, gen, d_in):
    n, hidden, c = 32, 2048, 9
    feats = torch.randn(n, d_in, device=dev, generator=gen).to(torch.bfloat16)
    w1 = (torch.randn(hidden, d_in, device=dev, generator=gen) / d_in ** 0.5).to(torch.bfloat16)
    b1 = torch.randn(hidden, device=dev, generator=gen) * 0.1
    w2 = (torch.randn(c, hidden, device=dev, generator=gen) / hidden ** 0.5).to(torch.bfloat16)
    b2 = torch.randn(c, device=dev, generator=gen) * 0.1
    cand = torch.arange(8, 8 + 2 * c, 2, dtype=torch.int32, device=dev)
    ws = bp.workspace(bp.policy_select_workspace_size(n, d_in, hidden, c), dev)
    return lambda: bp.policy_select(feats, w1, b1, w2, b2, cand, want_logits=False, ws=ws)


def _tau(dev, gen):
    n, j = 1 << 22, 24
    g = (0.86 + 0.05 * torch.randn(n, j, device=dev, generator=gen)).clamp_(0.05, 0.999).contiguous()
    cand = list(range(8, 25, 2))
    pred = torch.tensor(cand, dtype=torch.int32, device=dev)[torch.randint(0, len(cand), (n,), device=dev,
                                                                           generator=gen)].contiguous()
    ws = bp.workspace(bp.tau_select_workspace_size(n), dev)
    return lambda: bp.tau_select(g, cand, 16, 0.001, predicted=pred, ws=ws)


CASES = {
    "verify_epilogue_t1": lambda dev, gen: _verify_epilogue(dev, gen, 1.0),
    "verify_epilogue_t0": lambda dev, gen: _verify_epilogue(dev, gen, 0.0),
    "verify_stream_c5_t1": lambda dev, gen: _verify_stream_c5(dev, gen, 1.0),
    "verify_stream_c5_t0": lambda dev, gen: _verify_stream_c5(dev, gen, 0.0),
    "accept_t1": _accept,
    "accept_batch_t1": lambda dev, gen: _accept_batch(dev, gen, 1.0),
    "accept_batch_t0": lambda dev, gen: _accept_batch(dev, gen, 0.0),
    "attention": _attention,
    "attention_c3": lambda dev, gen: _batch_attention(dev, gen, *_ragged_shapes()),
    "attention_c5": lambda dev, gen: _batch_attention(dev, gen, [32768] * 8, [B] * 8),
    "accept_c5_t1": _accept_c5,
    "step_c5": _step_c5,
    "policy": lambda dev, gen: _policy(dev, gen, 2560),
    "policy_d151936": lambda dev, gen: _policy(dev, gen, V),
    "tau": _tau,
}


def main(argv=None) -> None:
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("case", choices=sorted(CASES))
    ap.add_argument("--calls", type=int, default=3)
    ap.add_argument("--warmup", type=int, default=2)
    ap.add_argument("--split", choices=["flat", "cluster"], default="flat")
    args = ap.parse_args(argv)
    SPLIT["split"] = args.split
    dev = torch.device("cuda:0")
    gen = torch.Generator(device=dev)
    gen.manual_seed(7)
    bp.load()
    call = CASES[args.case](dev, gen)
    for _ in range(args.warmup + args.calls):
        call()
    torch.cuda.synchronize(dev)
    print(f"{args.case}: {args.warmup} + {args.calls} calls done")


if __name__ == "__main__":
    main()
