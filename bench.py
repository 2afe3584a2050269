"""Benchmark of the block-verify hot path on GB300.

One step = one block-verify pass over the long-context batch (8 sequences, context 32768, block
B = 16, Qwen3-8B-shaped 32/8 heads, head_dim 128, bf16 KV; acceptance over a 151936-token vocabulary
at T = 1): bp_block_attention (causal within the block) followed by bp_spec_accept.  It is the
largest of the five workloads and the one whose bytes the kernels stream at scale.  Inputs are
seeded synthetic data already resident in HBM, drawn on the device with the workload's recipe; two
input copies of 1.23 GB each (far larger than the 129 MB L2) alternate, so no step finds its inputs
in L2.  Every timed step is one replay of a CUDA graph that holds exactly one step, and the steps
are timed with CUDA events on the launching stream.

The JSON line also carries: the roofline of the dominant kernel (the verify attention, timed alone,
live), the step's whole HBM roofline, every hot-path row timed on its own (among them the
Qwen3-4B-shaped batch-1 step, the ragged 32-request step, greedy acceptance, drafter attention, the
policy head and the next-row kernels), an end-to-end figure through the public API from pinned host
buffers, the CPU oracle's throughput on the host cores (all cores and one core) on a stated sample
of the same workload, and the SM clocks sampled during the timed region.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
Under torchrun each rank runs an independent replica on its own GPU (no data-path collective).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "verified tokens/sec and % of HBM roofline for block-verify attention+accept, 1 GB300"
HEADLINE = "long_context"   # 8 sequences x (32768 + 16) keys, T = 1
BATCH1 = "qwen3_4b"         # 1 sequence x (2048 + 16) keys: the batch-1 row
COPIES = 32                 # rotating input copies of the batch-1 rows (32 x 27.6 MB > L2)
L2_BYTES = 129e6


def headline_config(world: int) -> dict:
    """The workload the metric is measured on (the same dict in both arms of the benchmark)."""
    return {"workload": "long_context: 8 sequences, context 32768, block 16 (anchor + 15 drafts), 32/8 heads, "
                        "head_dim 128, bf16 KV; acceptance over vocab 151936 fp32 logits at T=1",
            "global_batch": 8 * world, "seq_len": 32784, "parallelism": f"replicas x{world}",
            "l2": "2 alternating input copies of 1227 MB each (> 129 MB L2)",
            "graph": "every timed step is one replay of a CUDA graph holding exactly one step"}


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def tensor_peak():
    """Sustained dense bf16 TFLOP/s (a kernel timed inside a long run), measured or the fallback."""
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        if "bf16_tflops_sustained" in d:
            return float(d["bf16_tflops_sustained"]), "measured"
    return 1700.0, "fallback"


def dist_env():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)), int(os.environ.get("LOCAL_RANK", 0))


def max_over_ranks(seconds: float, world: int, device=None) -> float:
    """The slowest rank's time: the job's time (every rank ran the same number of steps)."""
    if world <= 1:
        return seconds
    import torch
    import torch.distributed as dist

    t = torch.tensor([seconds], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(tokens_per_step: int, steps: int, seconds: float, world: int) -> float:
    """Whole-job tokens/s: every rank verifies tokens_per_step tokens per step (weak scaling)."""
    return world * tokens_per_step * steps / seconds


# ----------------------------------------------------------------------------- byte counts
def attention_bytes(w) -> float:
    """K and V read once, Q read and O written once (bf16)."""
    e = 2
    blocks = np.asarray(w.block)
    kv = (np.asarray(w.ctx) + blocks).sum() * w.num_kv_heads * w.head_dim * 2 * e
    qo = 2 * blocks.sum() * w.num_q_heads * w.head_dim * e
    return float(kv + qo)


def accept_bytes(w, temperature: float) -> float:
    """Target rows (gamma+1 per sequence) and, at T > 0, draft rows (gamma), fp32, read once."""
    g = np.asarray(w.block) - 1
    rows = (g + 1).sum() + (g.sum() if temperature > 0 else 0)
    return float(rows * w.vocab * 4)


def policy_bytes(pin) -> float:
    return float(pin["w1"].nbytes + pin["w2"].nbytes)


# ----------------------------------------------------------------------------- clocks
class ClockSampler:
    QUERY = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
             "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
             "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.QUERY}",
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.15)
        return self

    def __exit__(self, *exc):
        self.out = ""
        if self.proc is not None:
            time.sleep(0.1)
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.out, _ = self.proc.communicate()

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in (self.out or "").strip().splitlines():
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx = float(parts[1])
            except ValueError:
                continue
            for name, flag in zip(names, parts[4:8]):
                if flag.lower() == "active":
                    reasons.add(name)
        loaded = [x for x in sm if mx and x > 0.5 * mx] or sm
        return {"sm_mhz": statistics.median(loaded) if loaded else None, "sm_max_mhz": mx,
                "reasons": sorted(reasons), "samples": len(sm)}


# ----------------------------------------------------------------------------- our arm
def run_ours(args):
    import torch

    import paper_2606_31315_gb300 as bp
    from paper_2606_31315_gb300 import workloads as wl

    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    bp.build()
    bp.load()
    stream = torch.cuda.Stream(device=dev)
    peak, peak_kind = peaks()
    gen = torch.Generator(device=dev)
    gen.manual_seed(5)

    def t(x):
        return torch.from_numpy(np.ascontiguousarray(x)).to(dev)

    def bf(x):
        return torch.from_numpy(x.view(np.int16)).to(dev).view(torch.bfloat16)

    def graph_one(fn):
        """A CUDA graph holding exactly one call of fn (warmed outside the capture first)."""
        with torch.cuda.stream(stream):
            for _ in range(2):
                fn()
        stream.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            fn()
        stream.synchronize()
        return g

    def time_graph(g, reps):
        """Seconds per replay (events on the launching stream)."""
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize(dev)
        with torch.cuda.stream(stream):  # replay on the stream the events are recorded on
            e0.record(stream)
            for _ in range(reps):
                g.replay()
            e1.record(stream)
        e1.synchronize()
        return e0.elapsed_time(e1) / 1e3 / reps

    def time_alternating(gs, reps):
        """Seconds per replay of graphs gs[0], gs[1], ... in turn (one graph per input copy)."""
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize(dev)
        with torch.cuda.stream(stream):
            e0.record(stream)
            for i in range(reps):
                gs[i % len(gs)].replay()
            e1.record(stream)
        e1.synchronize()
        return e0.elapsed_time(e1) / 1e3 / reps

    def barrier():
        if world > 1:
            import torch.distributed as dist

            dist.barrier()

    def row(tsec, nbytes, kernels):
        gbs = nbytes / tsec / 1e9
        return {"us": round(tsec * 1e6, 3), "bytes": nbytes, "gbs": round(gbs, 1), "frac": round(gbs / peak, 4),
                "kernels": kernels}

    # ---------------- a batch workload's inputs, drawn on the device with the workload's recipe
    def batch_layout(sw):
        blocks = np.asarray(sw.block)
        kv = np.asarray(sw.ctx) + blocks
        gam = blocks - 1
        ns, ntd = sw.num_seqs, int(gam.sum())
        return dict(blocks=blocks, kv=kv, gam=gam, ns=ns, ntd=ntd, cu_q=t(wl.offsets(blocks)),
                    cu_kv=t(wl.offsets(kv)), cu_d=t(wl.offsets(gam)), max_q=int(blocks.max()), max_kv=int(kv.max()),
                    trow=t((np.arange(ntd) + np.repeat(np.arange(ns), gam)).astype(np.int64)))

    def draw_batch(sw, lay):
        """Q, K, V ~ N(0, 1) bf16; target logits ~ N(0, logit_std^2), draft = target + N(0, 1) fp32;
        T = 1 draft tokens by Gumbel-max over the draft row, T = 0 tokens its argmax; uniforms."""
        hd, hq, hkv = sw.head_dim, sw.num_q_heads, sw.num_kv_heads
        nq, nkv = int(lay["blocks"].sum()), int(lay["kv"].sum())
        c = dict(q=torch.randn(nq, hq, hd, device=dev, generator=gen).to(torch.bfloat16),
                 k=torch.randn(nkv, hkv, hd, device=dev, generator=gen).to(torch.bfloat16),
                 v=torch.randn(nkv, hkv, hd, device=dev, generator=gen).to(torch.bfloat16),
                 target=torch.randn(lay["ntd"] + lay["ns"], sw.vocab, device=dev, generator=gen) * sw.logit_std,
                 ua=torch.rand(lay["ntd"], device=dev, generator=gen), us=torch.rand(lay["ns"], device=dev,
                                                                                   generator=gen))
        c["o"] = torch.empty_like(c["q"])
        c["draft"] = c["target"][lay["trow"]] + torch.randn(lay["ntd"], sw.vocab, device=dev, generator=gen)
        ex = torch.empty_like(c["draft"]).exponential_(generator=gen)  # -log(E), E ~ Exp(1): Gumbel noise
        c["tok"] = torch.argmax(c["draft"] - torch.log(ex), dim=1).to(torch.int32)
        del ex
        c["tok0"] = torch.argmax(c["draft"], dim=1).to(torch.int32)
        return c

    class BatchStep:
        """Causal verify attention then the acceptance over a batch workload, on the caller's copies."""

        def __init__(self, sw, lay):
            self.sw, self.lay = sw, lay
            self.ws_at = bp.workspace(bp.block_attention_workspace_size(lay["ns"], lay["max_q"], sw.num_q_heads,
                                                                        sw.num_kv_heads, sw.head_dim), dev)
            self.ws_ac = bp.workspace(bp.spec_accept_workspace_size(lay["ns"], lay["ntd"], sw.vocab), dev)
            self.n = torch.empty(lay["ns"], dtype=torch.int32, device=dev)
            self.o = torch.empty(lay["ntd"] + lay["ns"], dtype=torch.int32, device=dev)

        def attn(self, c, mask=bp.MASK_CAUSAL):
            lay = self.lay
            bp.block_attention(c["q"], c["k"], c["v"], lay["cu_q"], lay["cu_kv"], lay["max_q"], lay["max_kv"],
                               mask=mask, out=c["o"], ws=self.ws_at, stream=stream)

        def accept(self, c, temp=1.0):
            lay = self.lay
            if temp > 0:
                bp.spec_accept(c["target"], c["draft"], c["tok"], lay["cu_d"], temp, c["ua"], c["us"],
                               n_accepted=self.n, out_tokens=self.o, want_accept_prob=False, ws=self.ws_ac,
                               stream=stream)
            else:
                bp.spec_accept(c["target"], None, c["tok0"], lay["cu_d"], 0.0, None, None, n_accepted=self.n,
                               out_tokens=self.o, want_accept_prob=False, ws=self.ws_ac, stream=stream)

        def step(self, c, temp=1.0):
            self.attn(c)
            self.accept(c, temp)

    # ================= the headline: the long-context verify step, K steps timed, one graph replay each
    hw = wl.get(HEADLINE)
    hlay = batch_layout(hw)
    hcopies = [draw_batch(hw, hlay) for _ in range(2)]
    hstep = BatchStep(hw, hlay)
    g_steps = [graph_one(lambda c=c: hstep.step(c)) for c in hcopies]
    with torch.cuda.stream(stream):
        for i in range(args.warmup):
            g_steps[i % 2].replay()
    stream.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    torch.cuda.synchronize(dev)
    with ClockSampler(local) as clk:
        with torch.cuda.stream(stream):
            e0.record(stream)
            for i in range(args.steps):
                g_steps[i % 2].replay()
            e1.record(stream)
        e1.synchronize()
    torch.cuda.synchronize(dev)
    barrier()
    elapsed = max_over_ranks(e0.elapsed_time(e1) / 1e3, world, dev)
    tokens_per_step = int(np.sum(hw.block))
    value = job_throughput(tokens_per_step, args.steps, elapsed, world)
    ms_per_step = elapsed / args.steps * 1e3
    step_bytes = attention_bytes(hw) + accept_bytes(hw, 1.0)
    # tokens the steps emit (the accepted drafts and one drawn token per sequence), on the two input copies
    emitted = []
    for g in g_steps:
        with torch.cuda.stream(stream):
            g.replay()
        stream.synchronize()
        emitted.append(int(hstep.n.sum().item()) + hw.num_seqs)
    emitted_per_step = float(np.mean(emitted))

    # the step's kernels timed alone (same alternation, graph replays): the dominant one is the attention
    reps_h = max(20, min(200, args.steps))
    t_h_attn = time_alternating([graph_one(lambda c=c: hstep.attn(c)) for c in hcopies], reps_h)
    t_h_acc1 = time_alternating([graph_one(lambda c=c: hstep.accept(c, 1.0)) for c in hcopies], reps_h)
    t_h_acc0 = time_alternating([graph_one(lambda c=c: hstep.accept(c, 0.0)) for c in hcopies], reps_h)
    t_h_step0 = time_alternating([graph_one(lambda c=c: hstep.step(c, 0.0)) for c in hcopies], reps_h)
    attn_h_bytes = attention_bytes(hw)
    roofline = {"bound": "hbm", "kernel": "attn_bf16_tc_kernel", "achieved": round(attn_h_bytes / t_h_attn / 1e9, 1),
                "peak": peak, "peak_kind": f"{peak_kind} hbm_gbs (burst copy)", "unit": "GB/s",
                "frac": round(attn_h_bytes / t_h_attn / 1e9 / peak, 4), "traffic": committed_traffic("attn_c5"),
                "algorithmic_bytes": attn_h_bytes, "avg_launch_us": round(t_h_attn * 1e6, 3),
                "per_unit": "K and V of (32768 + 16) keys x 8 KV heads x 128 x 2 B each, Q in and O out: "
                            "8 sequences per launch"}

    # end to end through the public API: every step copies its inputs from pinned host memory
    e2e = run_e2e(bp, torch, dev, stream, hw, hlay, hcopies[0], min(args.steps, 20))
    del g_steps, hcopies, hstep

    # ================= every other row, each timed alone
    # ---- batch 1, Qwen3-4B shapes: 32 rotating copies (882 MB > L2), graphs of 32 calls
    w = wl.get(BATCH1)
    a = wl.attention_inputs(w)
    acc = wl.accept_inputs(w, 1.0)
    acc0 = wl.accept_inputs(w, 0.0)
    copies = []
    for _ in range(COPIES):
        copies.append(dict(q=bf(a["q"]), k=bf(a["k"]), v=bf(a["v"]), o=torch.empty(a["q"].shape, dtype=torch.bfloat16,
                                                                                     device=dev),
                           target=t(acc["target_logits"]), draft=t(acc["draft_logits"]), tok=t(acc["draft_tokens"]),
                           ua=t(acc["u_accept"]), us=t(acc["u_sample"]), tok0=t(acc0["draft_tokens"])))
    cu_q, cu_kv, cu_d = t(a["cu_q"]), t(a["cu_kv"]), t(acc["cu_draft"])
    S, TD, V = w.num_seqs, int(acc["cu_draft"][-1]), w.vocab
    n_acc = torch.empty(S, dtype=torch.int32, device=dev)
    out_tok = torch.empty(TD + S, dtype=torch.int32, device=dev)
    ws_a = bp.workspace(bp.block_attention_workspace_size(S, a["max_q_len"], 32, 8, 128), dev)
    ws_s = bp.workspace(bp.spec_accept_workspace_size(S, TD, V), dev)

    def attn(c, mask=bp.MASK_CAUSAL):
        bp.block_attention(c["q"], c["k"], c["v"], cu_q, cu_kv, a["max_q_len"], a["max_kv_len"], mask=mask,
                           out=c["o"], ws=ws_a, stream=stream)

    def accept(c, temp=1.0):
        if temp > 0:
            bp.spec_accept(c["target"], c["draft"], c["tok"], cu_d, temp, c["ua"], c["us"], n_accepted=n_acc,
                           out_tokens=out_tok, want_accept_prob=False, ws=ws_s, stream=stream)
        else:
            bp.spec_accept(c["target"], None, c["tok0"], cu_d, 0.0, None, None, n_accepted=n_acc, out_tokens=out_tok,
                           want_accept_prob=False, ws=ws_s, stream=stream)

    def step(c):
        attn(c)
        accept(c)

    def graph_of(fn):
        """One CUDA graph running fn once on each input copy."""
        with torch.cuda.stream(stream):
            for c in copies:  # warm the code paths outside capture
                fn(c)
        stream.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for c in copies:
                fn(c)
        stream.synchronize()
        return g

    reps = 60
    t_step1 = time_graph(graph_of(step), reps) / COPIES
    t_attn = time_graph(graph_of(attn), reps) / COPIES
    t_acc = time_graph(graph_of(accept), reps) / COPIES
    t_bidir = time_graph(graph_of(lambda c: attn(c, bp.MASK_BIDIR)), reps) / COPIES
    t_acc0 = time_graph(graph_of(lambda c: accept(c, 0.0)), reps) / COPIES
    # next row: the same verify attention over a paged KV cache (64-row pages in shuffled order)
    page = 64
    pk = wl.paged_kv(a["k"], a["v"], a["cu_kv"], page, seed=1)
    for c in copies:
        c["kc"], c["vc"] = bf(pk["k_cache"]), bf(pk["v_cache"])
    bt = t(pk["block_table"])

    def attn_paged(c):
        bp.block_attention_paged(c["q"], c["kc"], c["vc"], cu_q, cu_kv, bt, page, int(a["cu_kv"][-1]),
                                 a["max_q_len"], a["max_kv_len"], out=c["o"], ws=ws_a, stream=stream)

    t_attn_paged = time_graph(graph_of(attn_paged), reps) / COPIES
    for c in copies:
        del c["kc"], c["vc"]
    pw = wl.get("ragged")
    pin = wl.policy_inputs(pw)
    for c in copies:  # one copy of the policy weights per input copy (32 x 10.5 MB > L2)
        c["pol"] = {k: (bf(pin[k]) if k in ("feats", "w1", "w2") else t(pin[k])) for k in
                    ("feats", "w1", "w2", "b1", "b2", "candidates", "row_index")}
    ws_p = bp.workspace(bp.policy_select_workspace_size(32, 2560, 2048, 9), dev)
    bsz = torch.empty(32, dtype=torch.int32, device=dev)

    def policy(c):
        pf = c["pol"]
        bp.policy_select(pf["feats"], pf["w1"], pf["b1"], pf["w2"], pf["b2"], pf["candidates"],
                         row_index=pf["row_index"], block_size=bsz, want_logits=False, ws=ws_p, stream=stream)

    t_pol = time_graph(graph_of(policy), reps) / COPIES

    def time_calls(fn, n_graph=4, reps=10):
        """Seconds per call: replays of a graph of n_graph calls, or timed eager calls if the launch
        cannot be captured."""
        with torch.cuda.stream(stream):
            for _ in range(3):
                fn(None)
        stream.synchronize()
        try:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                for _ in range(n_graph):
                    fn(None)
            return time_graph(g, reps) / n_graph
        except RuntimeError:
            torch.cuda.synchronize(dev)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            with torch.cuda.stream(stream):
                e0.record(stream)
                for _ in range(reps * n_graph):
                    fn(None)
                e1.record(stream)
            e1.synchronize()
            return e0.elapsed_time(e1) / 1e3 / (reps * n_graph)

    # next row: the policy head at the paper's own input width, d_in = V = 151936 (Section 3.1's
    # last-token logits); one seeded synthetic weight copy (622 MB, far larger than L2)
    big_n, big_d, big_h, big_c = 32, w.vocab, 2048, len(pin["candidates"])
    gen.manual_seed(7)
    big = dict(feats=torch.randn(big_n, big_d, device=dev, generator=gen).to(torch.bfloat16),
               w1=(torch.randn(big_h, big_d, device=dev, generator=gen) / big_d ** 0.5).to(torch.bfloat16),
               b1=torch.randn(big_h, device=dev, generator=gen) * 0.1,
               w2=(torch.randn(big_c, big_h, device=dev, generator=gen) / big_h ** 0.5).to(torch.bfloat16),
               b2=torch.randn(big_c, device=dev, generator=gen) * 0.1)
    ws_big = bp.workspace(bp.policy_select_workspace_size(big_n, big_d, big_h, big_c), dev)
    bsz_big = torch.empty(big_n, dtype=torch.int32, device=dev)
    cand_dev = t(pin["candidates"])

    def policy_big(_c):
        bp.policy_select(big["feats"], big["w1"], big["b1"], big["w2"], big["b2"], cand_dev, block_size=bsz_big,
                         want_logits=False, ws=ws_big, stream=stream)

    t_pol_big = time_calls(policy_big, n_graph=4, reps=10)
    big_bytes = float(big["w1"].numel() * 2 + big["feats"].numel() * 2 + big["w2"].numel() * 2)
    del big

    # next row: the LM head fused with the acceptance -- the Qwen3-4B LM head (151936 x 2560 bf16,
    # 778 MB, far larger than L2) over the batch-1 step's 16 target and 15 drafter states at T=1;
    # beside it the unfused path (cuBLAS bf16 GEMM to logits, fp32 cast, acceptance kernel)
    lm_h, td_q = 2560, int(w.block[0]) - 1
    w_lm = (torch.randn(w.vocab, lm_h, device=dev, generator=gen) * (w.logit_std / lm_h ** 0.5)).to(torch.bfloat16)
    h_t = torch.randn(td_q + 1, lm_h, device=dev, generator=gen).to(torch.bfloat16)
    h_d = (h_t[:td_q].float() + torch.randn(td_q, lm_h, device=dev, generator=gen) / w.logit_std).to(torch.bfloat16)
    ve_tok = torch.randint(0, w.vocab, (td_q,), device=dev, generator=gen, dtype=torch.int32)
    ve_cu = torch.tensor([0, td_q], dtype=torch.int32, device=dev)
    ve_ua, ve_us = torch.rand(td_q, device=dev, generator=gen), torch.rand(1, device=dev, generator=gen)
    ve_n, ve_o = torch.empty(1, dtype=torch.int32, device=dev), torch.empty(td_q + 1, dtype=torch.int32, device=dev)
    ws_ve = bp.workspace(bp.verify_epilogue_workspace_size(1, td_q, w.vocab), dev)

    def fused(_c):
        bp.verify_epilogue(w_lm, h_t, h_d, ve_tok, ve_cu, 1.0, ve_ua, ve_us, n_accepted=ve_n, out_tokens=ve_o,
                           want_accept_prob=False, ws=ws_ve, stream=stream)

    h_all = torch.cat([h_t, h_d])
    lg = torch.empty(2 * td_q + 1, w.vocab, dtype=torch.float32, device=dev)
    ws_u = bp.workspace(bp.spec_accept_workspace_size(1, td_q, w.vocab), dev)

    def unfused(_c):
        with torch.cuda.stream(stream):
            lg.copy_(torch.matmul(h_all, w_lm.t()))
        bp.spec_accept(lg[:td_q + 1], lg[td_q + 1:], ve_tok, ve_cu, 1.0, ve_ua, ve_us, n_accepted=ve_n,
                       out_tokens=ve_o, want_accept_prob=False, ws=ws_u, stream=stream)

    t_ve = time_calls(fused)
    t_unfused = time_calls(unfused)
    ve_bytes = float(w_lm.numel() * 2 + h_all.numel() * 2)
    del lg

    # next row: the same LM head over the long-context batch at T=1 -- 8 sequences x 16 positions, 128
    # target and 120 drafter states (248 rows: more logits than tensor memory holds, so the projection
    # streams and writes the logits once; the draw reads back only its row pairs) -- beside the unfused path
    lc = wl.get("long_context")
    S5, g5 = lc.num_seqs, int(lc.block[0]) - 1
    td5 = S5 * g5
    h5_t = torch.randn(td5 + S5, lm_h, device=dev, generator=gen).to(torch.bfloat16)
    trow5 = torch.arange(td5, device=dev) + torch.arange(td5, device=dev) // g5  # target row of draft i
    h5_d = (h5_t[trow5].float() + torch.randn(td5, lm_h, device=dev, generator=gen) / lc.logit_std).to(torch.bfloat16)
    tok5 = torch.randint(0, lc.vocab, (td5,), device=dev, generator=gen, dtype=torch.int32)
    cu5 = torch.arange(0, td5 + 1, g5, dtype=torch.int32, device=dev)
    ua5, us5 = torch.rand(td5, device=dev, generator=gen), torch.rand(S5, device=dev, generator=gen)
    n5, o5 = torch.empty(S5, dtype=torch.int32, device=dev), torch.empty(td5 + S5, dtype=torch.int32, device=dev)
    ws_ve5 = bp.workspace(bp.verify_epilogue_workspace_size(S5, td5, lc.vocab), dev)

    def fused5(_c):
        bp.verify_epilogue(w_lm, h5_t, h5_d, tok5, cu5, 1.0, ua5, us5, n_accepted=n5, out_tokens=o5,
                           want_accept_prob=False, ws=ws_ve5, stream=stream)

    h5_all = torch.cat([h5_t, h5_d])
    lg5 = torch.empty(h5_all.shape[0], lc.vocab, dtype=torch.float32, device=dev)
    ws_u5 = bp.workspace(bp.spec_accept_workspace_size(S5, td5, lc.vocab), dev)

    def unfused5(_c):
        with torch.cuda.stream(stream):
            lg5.copy_(torch.matmul(h5_all, w_lm.t()))
        bp.spec_accept(lg5[:td5 + S5], lg5[td5 + S5:], tok5, cu5, 1.0, ua5, us5, n_accepted=n5, out_tokens=o5,
                       want_accept_prob=False, ws=ws_u5, stream=stream)

    t_ve5 = time_calls(fused5)
    t_unfused5 = time_calls(unfused5)
    rows5 = h5_all.shape[0]
    ve5_bytes = float(w_lm.numel() * 2 + h5_all.numel() * 2)  # the operation's own operands
    ve5_hbm = ve5_bytes + rows5 * lc.vocab * 4.0 + 2 * S5 * lc.vocab * 4.0  # + logits written, draw pairs read
    ve5_flops = 2.0 * rows5 * lc.vocab * lm_h
    del w_lm, lg5, ws_ve5, ws_u5

    # next row: the decoding loop on the device -- each step runs 36 layers (Qwen3-4B) of append-the-block
    # + paged verify attention, the T=1 acceptance and the commit (lengths back to the accepted prefix,
    # next offsets on the device); a graph of 8 steps that starts by resetting the lengths, replayed
    n_layers, loop_steps_n, page_l = 36, 8, 64
    ctx0, blk = int(w.ctx[0]), int(w.block[0])
    cap_l = -(-(ctx0 + (loop_steps_n + 1) * blk) // page_l) * page_l
    pps_l = cap_l // page_l
    pool_k = [torch.randn(cap_l, w.num_kv_heads, w.head_dim, device=dev, generator=gen).to(torch.bfloat16)
              for _ in range(n_layers)]
    pool_v = [torch.randn(cap_l, w.num_kv_heads, w.head_dim, device=dev, generator=gen).to(torch.bfloat16)
              for _ in range(n_layers)]
    bt_l = torch.arange(pps_l, dtype=torch.int32, device=dev).view(1, pps_l)
    kn_l = torch.randn(blk, w.num_kv_heads, w.head_dim, device=dev, generator=gen).to(torch.bfloat16)
    vn_l = torch.randn(blk, w.num_kv_heads, w.head_dim, device=dev, generator=gen).to(torch.bfloat16)
    o_l = torch.empty(blk, w.num_q_heads, w.head_dim, dtype=torch.bfloat16, device=dev)
    cu_q_l = torch.tensor([0, blk], dtype=torch.int32, device=dev)
    ctx_init = torch.tensor([ctx0], dtype=torch.int32, device=dev)
    cu_kv_init = torch.tensor([0, ctx0 + blk], dtype=torch.int32, device=dev)
    ctx_d, cu_kv_d = ctx_init.clone(), cu_kv_init.clone()
    na_l, ot_l = torch.empty(1, dtype=torch.int32, device=dev), torch.empty(blk, dtype=torch.int32, device=dev)
    anc_l = torch.empty(1, dtype=torch.int32, device=dev)
    ws_acc_l = bp.workspace(bp.spec_accept_workspace_size(1, blk - 1, w.vocab), dev)
    ws_c = bp.workspace(256, dev)
    c0_ = copies[0]

    def loop_steps(_c):
        with torch.cuda.stream(stream):
            ctx_d.copy_(ctx_init)
            cu_kv_d.copy_(cu_kv_init)
        for _ in range(loop_steps_n):
            for l in range(n_layers):
                bp.kv_append(pool_k[l], pool_v[l], kn_l, vn_l, cu_q_l, cu_kv_d, bt_l, page_l, stream=stream)
                bp.block_attention_paged(c0_["q"], pool_k[l], pool_v[l], cu_q_l, cu_kv_d, bt_l, page_l, cap_l, blk,
                                         cap_l, out=o_l, ws=ws_a, stream=stream)
            bp.spec_accept(c0_["target"], c0_["draft"], c0_["tok"], cu_d, 1.0, c0_["ua"], c0_["us"], n_accepted=na_l,
                           out_tokens=ot_l, want_accept_prob=False, ws=ws_acc_l, stream=stream)
            bp.verify_commit(ctx_d, na_l, ot_l, cu_d, cap_l, anchor=anc_l, cu_kv_next=cu_kv_d, ws=ws_c, stream=stream)

    t_loop = time_calls(loop_steps, n_graph=1, reps=10) / loop_steps_n
    loop_bytes = n_layers * (attention_bytes(w) + 2 * kn_l.numel() * 2 * 2) + accept_bytes(w, 1.0)
    del pool_k, pool_v

    # next row: Appendix A's acceptance-length model over 4M requests (24 positions each, the nine
    # candidate sizes): tau per candidate, B*, regret of a predicted size, the bound's summary
    n_tau, j_tau = 1 << 22, 24
    torch.manual_seed(8)  # the Beta sampler draws from the global generator
    gx = torch.distributions.Beta(torch.tensor(12.0, device=dev), torch.tensor(2.0, device=dev)).sample((n_tau, 1))
    g_tau = (gx + 0.03 * torch.randn(n_tau, j_tau, device=dev, generator=gen)).clamp_(0.05, 0.999).contiguous()
    cand_tau = wl.CANDIDATES  # host array
    pred_tau = t(wl.CANDIDATES)[torch.randint(0, len(wl.CANDIDATES), (n_tau,), device=dev, generator=gen)].contiguous()
    tau_out = torch.empty(n_tau, len(wl.CANDIDATES), device=dev)
    best_tau = torch.empty(n_tau, dtype=torch.int32, device=dev)
    reg_tau = torch.empty(n_tau, device=dev)
    sum_tau = torch.empty(4, dtype=torch.float64, device=dev)
    ws_tau = bp.workspace(bp.tau_select_workspace_size(n_tau), dev)

    def tau_model(_c):
        bp.tau_select(g_tau, cand_tau, 16, 0.001, predicted=pred_tau, tau=tau_out, best=best_tau, regret=reg_tau,
                      summary=sum_tau, ws=ws_tau, stream=stream)

    t_tau = time_calls(tau_model, n_graph=4, reps=20)
    tau_bytes = float(g_tau.numel() * 4 + pred_tau.numel() * 4 + tau_out.numel() * 4 + best_tau.numel() * 4
                      + reg_tau.numel() * 4)
    del g_tau, tau_out

    # a5-a7 at batch scale: the 32-request ragged batch (blocks 8..24: 502 target and 470 drafter rows
    # over the 151936-token vocabulary), which runs the three throughput kernels; 2 alternating copies
    rw = wl.get("ragged")
    rlay = batch_layout(rw)
    rcopies = [draw_batch(rw, rlay) for _ in range(2)]
    rstep = BatchStep(rw, rlay)
    t_racc1 = time_alternating([graph_one(lambda c=c: rstep.accept(c, 1.0)) for c in rcopies], 20)
    t_racc0 = time_alternating([graph_one(lambda c=c: rstep.accept(c, 0.0)) for c in rcopies], 20)
    t_rattn = time_alternating([graph_one(lambda c=c: rstep.attn(c)) for c in rcopies], 20)
    t_rstep = time_alternating([graph_one(lambda c=c: rstep.step(c)) for c in rcopies], 20)
    del rcopies, rstep

    # a3 at the drafter's own configuration: 16 sequences of 4096 context keys and a 16-position block of
    # mask-token queries, bidirectional within the block (269 MB of K/V, larger than L2), drawn on the device
    dw = wl.get("drafter_bidir")
    d_kv = np.asarray(dw.ctx) + np.asarray(dw.block)
    d_cu_q, d_cu_kv = t(wl.offsets(dw.block)), t(wl.offsets(d_kv))
    d_q = torch.randn(int(np.sum(dw.block)), dw.num_q_heads, dw.head_dim, device=dev, generator=gen).to(torch.bfloat16)
    d_k = torch.randn(int(d_kv.sum()), dw.num_kv_heads, dw.head_dim, device=dev, generator=gen).to(torch.bfloat16)
    d_v = torch.randn(int(d_kv.sum()), dw.num_kv_heads, dw.head_dim, device=dev, generator=gen).to(torch.bfloat16)
    d_o = torch.empty_like(d_q)
    ws_d = bp.workspace(bp.block_attention_workspace_size(dw.num_seqs, int(max(dw.block)), dw.num_q_heads,
                                                          dw.num_kv_heads, dw.head_dim), dev)

    def drafter_attn(_c):
        bp.block_attention(d_q, d_k, d_v, d_cu_q, d_cu_kv, int(max(dw.block)), int(d_kv.max()), mask=bp.MASK_BIDIR,
                           out=d_o, ws=ws_d, stream=stream)

    t_drafter = time_calls(drafter_attn, n_graph=4, reps=10)
    del d_q, d_k, d_v, d_o

    def step_row(tsec, sw, temp, kernels, what):
        nbytes = attention_bytes(sw) + accept_bytes(sw, temp)
        tokens = int(np.sum(sw.block))
        out = row(tsec, nbytes, kernels)
        out.update(verified_tokens_per_s=round(tokens / tsec, 1), requests_per_s=round(sw.num_seqs / tsec, 1),
                   roofline_tokens_per_s=round(tokens / (nbytes / (peak * 1e9)), 1), workload=what)
        return out

    batch_kernels1 = ["batch_stats_kernel<false,true>", "batch_draw_kernel (decisions inside)"]
    batch_kernels0 = ["batch_stats_kernel<true,true>", "batch_decide_kernel"]
    rows = {
        "c5_attention_causal_8x32784": dict(row(t_h_attn, attn_h_bytes, ["attn_bf16_tc_kernel (flat split)",
                                                                         "attn_combine_kernel"]),
                                            traffic=committed_traffic("attn_c5")),
        "c5_accept_t1_8x16": row(t_h_acc1, accept_bytes(hw, 1.0), batch_kernels1),
        "c5_accept_greedy_t0_8x16": row(t_h_acc0, accept_bytes(hw, 0.0), batch_kernels0),
        "c5_step_t0_attention_accept_greedy": step_row(t_h_step0, hw, 0.0,
                                                       ["attn_bf16_tc_kernel (flat split)", "attn_combine_kernel"]
                                                       + batch_kernels0,
                                                       "8 sequences x (32768 + 16) keys, greedy acceptance"),
        "c3_step_ragged_32req_attention_accept_t1": step_row(
            t_rstep, rw, 1.0, ["attn_bf16_tc_kernel"] + batch_kernels1,
            f"32 sequences, {int(np.sum(rw.block))} block positions, contexts {min(rw.ctx)}-{max(rw.ctx)}, "
            f"vocab {rw.vocab}, T=1"),
        "c3_attention_causal_ragged_32req": dict(row(t_rattn, attention_bytes(rw), ["attn_bf16_tc_kernel"]),
                                                 traffic=committed_traffic("attn_c3")),
        "a5_a6_accept_t1_batch_ragged_32req": dict(row(t_racc1, accept_bytes(rw, 1.0), batch_kernels1),
                                                   traffic=committed_traffic("batch_stats_kernel")),
        "a7_accept_greedy_t0_batch_ragged_32req": row(t_racc0, accept_bytes(rw, 0.0), batch_kernels0),
        "c2_step_qwen3_4b_batch1_attention_accept_t1": step_row(
            t_step1, w, 1.0, ["attn_bf16_tc_kernel", "accept_kernel<false,true>"],
            "1 sequence x (2048 + 16) keys, Qwen3-4B heads, vocab 151936, T=1 (graphs of 32 steps over 32 copies)"),
        "a2_a4_verify_attention_causal_qwen3_4b": dict(row(t_attn, attention_bytes(w), ["attn_bf16_tc_kernel"]),
                                                       traffic=committed_traffic("attn_c2")),
        "a3_drafter_attention_bidir_qwen3_4b": row(t_bidir, attention_bytes(w), ["attn_bf16_tc_kernel"]),
        "a3_drafter_attention_bidir_16x4112": row(t_drafter, attention_bytes(dw), ["attn_bf16_tc_kernel"]),
        "a5_a6_accept_t1_qwen3_4b": dict(row(t_acc, accept_bytes(w, 1.0), ["accept_kernel<false,true>"]),
                                         traffic=committed_traffic("accept_kernel")),
        "a7_accept_greedy_t0_qwen3_4b": row(t_acc0, accept_bytes(w, 0.0), ["accept_kernel<true,true>"]),
        "a1_policy_head_32req_2560x2048": row(t_pol, policy_bytes(pin), ["policy_tc_kernel"]),
        "next3_verify_attention_paged_page64": row(t_attn_paged, attention_bytes(w), ["attn_bf16_tc_kernel (paged)"]),
        "next2_policy_head_32req_151936x2048": dict(
            row(t_pol_big, big_bytes, ["policy_gather_kernel", "policy_tc_kernel<true,5> (streamed)"]),
            traffic=committed_traffic("policy_tc_kernel_ring")),
        "next1_fused_verify_epilogue_qwen3_4b_t1": dict(
            row(t_ve, ve_bytes, ["verify_epilogue_kernel<false,32,2>"]),
            traffic=committed_traffic("verify_epilogue_kernel"),
            unfused_us=round(t_unfused * 1e6, 3),
            unfused="cuBLAS bf16 GEMM to logits + fp32 cast + accept_kernel"),
        "next1_fused_verify_epilogue_long_context_t1": dict(
            row(t_ve5, ve5_bytes, ["lm_head_stream_kernel<false,2,true>", "lm_head_row_merge_kernel",
                                   "batch_draw_kernel"]),
            traffic=committed_traffic("lm_head_stream_kernel"),
            rows=int(rows5), design_hbm_bytes=ve5_hbm,
            design_frac=round(ve5_hbm / t_ve5 / 1e9 / peak, 4),
            tflops=round(ve5_flops / t_ve5 / 1e12, 1),
            tensor_frac=round(ve5_flops / t_ve5 / 1e12 / tensor_peak()[0], 4),
            unfused_us=round(t_unfused5 * 1e6, 3),
            unfused="cuBLAS bf16 GEMM to logits + fp32 cast + the throughput acceptance (statistics, draw)"),
        "next3_verify_loop_step_qwen3_4b_36_layers": dict(
            row(t_loop, loop_bytes, ["kv_append_kernel", "attn_bf16_tc_kernel (paged)", "accept_kernel<false,true>",
                                     "verify_commit_kernel"]),
            per_step="36 x (append + paged verify attention, 64-row pages) + T=1 acceptance + commit; the "
                     "context grows from 2048 by the accepted prefix each step; bytes counted at 2048 + 16 keys"),
        "next4_tau_model_4M_requests": dict(row(t_tau, tau_bytes, ["tau_kernel<24,9>", "tau_finish_kernel"]),
                                            traffic=committed_traffic("tau_kernel")),
    }

    result = {
        "metric": METRIC, "value": round(value, 1), "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms_per_step, 6), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": headline_config(world),
        "hbm_roofline": {"step_bytes": step_bytes, "achieved_gbs": round(step_bytes / (elapsed / args.steps) / 1e9, 1),
                         "peak": peak, "frac": round(step_bytes / (elapsed / args.steps) / 1e9 / peak, 4),
                         "roofline_tokens_per_s": round(tokens_per_step / (step_bytes / (peak * 1e9)), 1),
                         "requests_per_s": round(job_throughput(hw.num_seqs, args.steps, elapsed, world), 1),
                         "emitted_tokens_per_s": round(emitted_per_step * args.steps * world / elapsed, 1),
                         "emitted_per_step": emitted_per_step,
                         "roofline_requests_per_s": round(hw.num_seqs / (step_bytes / (peak * 1e9)), 1)},
        "roofline": roofline,
        "rows": rows,
        "e2e": e2e,
        "gpu_launches": STEP_LAUNCHES * args.steps,
        "gpu_launches_per_step": STEP_KERNELS,
        "clocks": clk.summary(),
    }
    if rank == 0:
        result["cpu_baseline"] = cpu_baseline(seconds=args.cpu_seconds)
        print(json.dumps(result), flush=True)
    if world > 1:
        import torch.distributed as dist

        dist.destroy_process_group()


# The kernels one headline step launches: the verify attention (its flat split and the merge of the cut
# units: 8 x 32784 keys leave the cluster split's SMs idle), then the acceptance's two throughput kernels
# (the T = 1 acceptance of 8 x 31 rows reads 37.7M logits, past the 6.5M crossover; the draw kernel takes
# the decisions).
STEP_KERNELS = ["attn_bf16_tc_kernel", "attn_combine_kernel", "batch_stats_kernel", "batch_draw_kernel"]
STEP_LAUNCHES = len(STEP_KERNELS)


def committed_traffic(kernel: str):
    """DRAM bytes per launch from the committed ncu summary, if it was taken on the current source."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        d = json.load(f).get(kernel)
    if not d:
        return None
    src = os.path.join(ROOT, "paper_2606_31315_gb300", "csrc", d["source"])
    with open(src, "rb") as f:
        digest = hashlib.sha256(f.read()).hexdigest()[:16]
    return d["dram_bytes_per_launch"] if digest == d["source_sha256_16"] else None


def run_e2e(bp, torch, dev, stream, sw, lay, c_dev, steps):
    """The same metric through the public API with the inputs in pinned host memory: every step copies
    its inputs host->device, runs both calls and copies the emitted tokens and accepted counts back.
    The copies run on their own stream into double-buffered device inputs, so step i+1's copies overlap
    step i's kernels; each step's kernels wait for its own copies, and every copy is inside the timed
    region."""
    keys = ("q", "k", "v", "target", "draft", "tok", "ua", "us")
    host = {k: c_dev[k].cpu().pin_memory() for k in keys}
    for k, x in (("cu_q", lay["cu_q"]), ("cu_kv", lay["cu_kv"]), ("cu_d", lay["cu_d"])):
        host[k] = x.cpu().pin_memory()
    sets = [{k: torch.empty_like(v, device=dev) for k, v in host.items()} for _ in range(2)]
    S, TD = lay["ns"], lay["ntd"]
    out_h = torch.empty(TD + S, dtype=torch.int32).pin_memory()
    nacc_h = torch.empty(S, dtype=torch.int32).pin_memory()
    n_acc = torch.empty(S, dtype=torch.int32, device=dev)
    out_tok = torch.empty(TD + S, dtype=torch.int32, device=dev)
    o = torch.empty_like(c_dev["q"])
    ws_a = bp.workspace(bp.block_attention_workspace_size(S, lay["max_q"], sw.num_q_heads, sw.num_kv_heads,
                                                          sw.head_dim), dev)
    ws_s = bp.workspace(bp.spec_accept_workspace_size(S, TD, sw.vocab), dev)
    h2d = sum(v.numel() * v.element_size() for v in host.values())
    d2h = out_h.numel() * 4 + nacc_h.numel() * 4
    copy_stream = torch.cuda.Stream(device=dev)
    freed = [torch.cuda.Event() for _ in range(2)]  # the kernels of the set's previous step are done

    def one(i):
        dv = sets[i % 2]
        copy_stream.wait_event(freed[i % 2])
        with torch.cuda.stream(copy_stream):
            for k, v in host.items():
                dv[k].copy_(v, non_blocking=True)
        copied = torch.cuda.Event()
        copied.record(copy_stream)
        stream.wait_event(copied)
        with torch.cuda.stream(stream):
            bp.block_attention(dv["q"], dv["k"], dv["v"], dv["cu_q"], dv["cu_kv"], lay["max_q"], lay["max_kv"], out=o,
                               ws=ws_a, stream=stream)
            bp.spec_accept(dv["target"], dv["draft"], dv["tok"], dv["cu_d"], 1.0, dv["ua"], dv["us"],
                           n_accepted=n_acc, out_tokens=out_tok, want_accept_prob=False, ws=ws_s, stream=stream)
            out_h.copy_(out_tok, non_blocking=True)
            nacc_h.copy_(n_acc, non_blocking=True)
        freed[i % 2].record(stream)

    for e in freed:
        e.record(stream)
    for i in range(3):
        one(i)
    torch.cuda.synchronize(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for e in freed:  # the timed copies start after e0
        e.record(stream)
    for i in range(steps):
        one(i)
    e1.record(stream)
    e1.synchronize()
    sec = e0.elapsed_time(e1) / 1e3 / steps
    del sets, host
    return {"value": round(int(np.sum(sw.block)) / sec, 1), "unit": "tokens/s", "h2d_bytes_per_step": int(h2d),
            "d2h_bytes_per_step": int(d2h), "steps": steps, "ms_per_step": round(sec * 1e3, 4),
            "host_link_gbs": round(h2d / sec / 1e9, 1),
            "copies": "one copy stream, double-buffered device inputs, overlapping the previous step's kernels"}


# ----------------------------------------------------------------------------- CPU oracle
def oracle_sample_fn():
    """One sequence of the long-context workload (context 32768, block 16, 32/8 heads, vocab 151936,
    T = 1), drawn by the workload module: the oracle's attention over all heads and its acceptance.
    A full step is 8 such sequences; the sample's throughput is its 16 verified tokens over its time."""
    import oracle
    from paper_2606_31315_gb300 import workloads as wl

    oracle.build()
    hw = wl.get(HEADLINE)
    w1 = wl.custom(name="long_context_1seq", seed=hw.seed, ctx=hw.ctx[:1], block=hw.block[:1],
                   num_q_heads=hw.num_q_heads, num_kv_heads=hw.num_kv_heads, head_dim=hw.head_dim, dtype=hw.dtype,
                   vocab=hw.vocab, logit_std=hw.logit_std, temperatures=(1.0,))
    a = wl.attention_inputs(w1)
    acc = wl.accept_inputs(w1, 1.0)
    q, k, v = (wl.as_f64(a[x], "bf16") for x in ("q", "k", "v"))
    g = w1.num_q_heads // w1.num_kv_heads

    def sample(kv_heads=None):
        """The sample's attention (all KV heads, or the first kv_heads of them: none for 0) and its
        acceptance."""
        if kv_heads is None:
            oracle.block_attention(q, k, v, a["cu_q"], a["cu_kv"], w1.num_kv_heads, oracle.MASK_CAUSAL)
        elif kv_heads > 0:
            oracle.block_attention(q[:, :kv_heads * g], k[:, :kv_heads], v[:, :kv_heads], a["cu_q"], a["cu_kv"],
                                   kv_heads, oracle.MASK_CAUSAL)
        oracle.spec_accept(acc["target_logits"], acc["draft_logits"], acc["draft_tokens"], acc["cu_draft"], 1.0,
                           acc["u_accept"], acc["u_sample"])

    return sample, int(np.sum(w1.block)), w1.num_kv_heads


def cpu_baseline(seconds: float = 10.0):
    """The fp64 oracle, as it stands, on the host cores: whole one-sequence samples of the long-context
    workload on all cores for a bounded time; on one core, the attention of one KV head (of 8) plus
    the sequence's acceptance, the attention time scaled by 8."""
    import oracle

    sample, tokens, hkv = oracle_sample_fn()
    cores = len(os.sched_getaffinity(0))
    oracle.set_num_threads(cores)
    sample()  # the first call pays for page faults
    n, t0 = 0, time.perf_counter()
    while True:
        sample()
        n += 1
        el = time.perf_counter() - t0
        if el >= seconds:
            break
    all_cores = tokens * n / el
    oracle.set_num_threads(1)
    t1 = time.perf_counter()
    sample(kv_heads=1)
    t_one = time.perf_counter() - t1
    t2 = time.perf_counter()
    sample(kv_heads=0)  # the acceptance alone (no attention heads)
    t_acc = time.perf_counter() - t2
    oracle.set_num_threads(cores)
    single = tokens / ((t_one - t_acc) * hkv + t_acc)
    return {"value": round(all_cores, 2), "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "sample": f"{n} one-sequence samples of long_context (causal attention over 32784 keys x 32 heads + "
                      f"T=1 acceptance of 31 rows x 151936; 16 verified tokens each) in {el:.1f} s on {cores} cores; "
                      f"a full step is 8 such sequences",
            "single_core": {"value": round(single, 3), "unit": "tokens/s", "cores": 1,
                            "sample": f"attention of 1 of 8 KV heads ({t_one - t_acc:.2f} s, scaled x8) + the "
                                      f"sequence's acceptance ({t_acc:.2f} s) on one thread"}}


def run_reference(args):
    """The reference arm: the oracle on the host cores, on the headline workload.  Each step is a
    bounded sample -- one of the workload's 8 sequences -- and the throughput is its verified tokens
    over its time."""
    rank, world, _ = dist_env()
    if rank != 0:
        return
    import oracle

    sample, tokens, _ = oracle_sample_fn()
    cores = len(os.sched_getaffinity(0))
    oracle.set_num_threads(cores)
    for _ in range(args.warmup):
        sample()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        sample()
    el = time.perf_counter() - t0
    value = tokens * args.steps / el
    res = {"impl": "reference", "metric": METRIC, "value": round(value, 2), "unit": "tokens/s", "n_gpus": world,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(el / args.steps * 1e3, 3),
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "config": headline_config(world),
           "cpu_baseline": {"value": round(value, 2), "unit": "tokens/s", "cores": cores, "kind": "oracle",
                            "sample": f"each step one of long_context's 8 sequences (causal attention over 32784 "
                                      f"keys x 32 heads + T=1 acceptance of 31 rows x 151936), {args.steps} steps "
                                      f"on {cores} host cores"},
           "e2e": {"value": round(value, 2), "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(res), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None)
    ap.add_argument("--warmup", type=int, default=None)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    args = ap.parse_args()
    if args.impl == "reference":
        args.steps = 20 if args.steps is None else args.steps
        args.warmup = 3 if args.warmup is None else args.warmup
        run_reference(args)
    else:
        args.steps = 2000 if args.steps is None else args.steps
        args.warmup = 50 if args.warmup is None else max(3, args.warmup)
        run_ours(args)


if __name__ == "__main__":
    main()
