"""GPU parity of the decoding loop with device-side rollback: every step appends each layer's block
K/V to a paged cache (bp_kv_append), runs the verify attention over it (bp_block_attention_paged),
accepts (bp_spec_accept, greedy) and commits (bp_verify_commit: the lengths fall back to anchor +
accepted drafts, the next offsets and anchors are written on the device).  The steps run eagerly and
again captured in one CUDA graph; an fp64 oracle loop keeps each sequence's cache rows as lists.

Bars: attention per (sequence, query head) within 2e-2 of max|O_ref| (the attention bar); n_accepted,
anchors, lengths, offsets and the retained cache rows bit-exact (greedy decisions on identical fp32
logits; the cache holds copied bf16 bytes)."""
import numpy as np
import pytest
import torch

import oracle
import paper_2606_31315_gb300 as bp
from paper_2606_31315_gb300 import workloads as wl

from _gpu import dev, to_dev

pytestmark = pytest.mark.gpu

BLOCKS = (8, 5, 16)
CTX = (100, 37, 260)
LAYERS, STEPS, HQ, HKV, D, PAGE, V = 2, 4, 8, 2, 128, 16, 1000


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    bp.build()
    bp.load()


def make_inputs(seed=5):
    rng = np.random.default_rng(seed)
    S = len(BLOCKS)
    gam = np.array(BLOCKS) - 1
    cu_draft = wl.offsets(gam)
    td = int(cu_draft[-1])
    nb = int(sum(BLOCKS))
    cap = -(-(max(CTX) + (STEPS + 1) * max(BLOCKS)) // PAGE) * PAGE
    bits = lambda *shape: wl.f32_to_bf16_bits(rng.standard_normal(shape, dtype=np.float32))  # noqa: E731
    ctx_k = [bits(sum(CTX), HKV, D) for _ in range(LAYERS)]
    ctx_v = [bits(sum(CTX), HKV, D) for _ in range(LAYERS)]
    q = [[bits(nb, HQ, D) for _ in range(LAYERS)] for _ in range(STEPS)]
    kn = [[bits(nb, HKV, D) for _ in range(LAYERS)] for _ in range(STEPS)]
    vn = [[bits(nb, HKV, D) for _ in range(LAYERS)] for _ in range(STEPS)]
    tokens, target = [], []
    seq_of = np.repeat(np.arange(S), gam)
    for _ in range(STEPS):
        tok = rng.integers(0, V, size=td).astype(np.int32)
        t = rng.standard_normal((td + S, V)).astype(np.float32) * 3
        agree = rng.random(td) < 0.75  # the target's argmax is the draft at these positions
        t[np.arange(td)[agree] + seq_of[agree], tok[agree]] = 30.0
        tokens.append(tok)
        target.append(t)
    return dict(cu_draft=cu_draft, cap=cap, ctx_k=ctx_k, ctx_v=ctx_v, q=q, kn=kn, vn=vn, tokens=tokens, target=target)


def setup_device(inp):
    """Paged pools holding the contexts (capacity rows per sequence, context rows filled)."""
    S, cap = len(BLOCKS), inp["cap"]
    cu_full = wl.offsets([cap] * S)
    pools = []
    for l in range(LAYERS):
        kf = np.zeros((S * cap, HKV, D), dtype=np.uint16)
        vf = np.zeros_like(kf)
        c0 = wl.offsets(CTX)
        for s in range(S):
            kf[s * cap:s * cap + CTX[s]] = inp["ctx_k"][l][c0[s]:c0[s + 1]]
            vf[s * cap:s * cap + CTX[s]] = inp["ctx_v"][l][c0[s]:c0[s + 1]]
        pools.append(wl.paged_kv(kf, vf, cu_full, PAGE, seed=11 + l, rows_per_seq=CTX))  # its own page order
    return pools


def run_loop(inp, pools, graph: bool):
    S = len(BLOCKS)
    cu_q = to_dev(wl.offsets(BLOCKS))
    cu_draft = to_dev(inp["cu_draft"])
    ctx = to_dev(np.array(CTX, dtype=np.int32))
    cu_kv = to_dev(wl.offsets(np.array(CTX) + np.array(BLOCKS)))
    kc = [to_dev(pl["k_cache"], "bf16") for pl in pools]
    vc = [to_dev(pl["v_cache"], "bf16") for pl in pools]
    bts = [to_dev(pl["block_table"]) for pl in pools]
    q = [[to_dev(x, "bf16") for x in st] for st in inp["q"]]
    kn = [[to_dev(x, "bf16") for x in st] for st in inp["kn"]]
    vn = [[to_dev(x, "bf16") for x in st] for st in inp["vn"]]
    tgt = [to_dev(t) for t in inp["target"]]
    tok = [to_dev(t) for t in inp["tokens"]]
    td = int(inp["cu_draft"][-1])
    nb = int(sum(BLOCKS))
    o = [[torch.empty(nb, HQ, D, dtype=torch.bfloat16, device=dev()) for _ in range(LAYERS)] for _ in range(STEPS)]
    nacc = [torch.empty(S, dtype=torch.int32, device=dev()) for _ in range(STEPS)]
    out = [torch.empty(td + S, dtype=torch.int32, device=dev()) for _ in range(STEPS)]
    anchor = [torch.empty(S, dtype=torch.int32, device=dev()) for _ in range(STEPS)]
    ws_a = [bp.workspace(bp.block_attention_workspace_size(S, max(BLOCKS), HQ, HKV, D), dev()) for _ in range(LAYERS)]
    ws_acc = bp.workspace(bp.spec_accept_workspace_size(S, td, V), dev())
    ws_c = bp.workspace(256, dev())
    stream = torch.cuda.Stream(dev())
    cap = inp["cap"]

    def loop():
        for st in range(STEPS):
            for l in range(LAYERS):
                bp.kv_append(kc[l], vc[l], kn[st][l], vn[st][l], cu_q, cu_kv, bts[l], PAGE, stream=stream)
                bp.block_attention_paged(q[st][l], kc[l], vc[l], cu_q, cu_kv, bts[l], PAGE, S * cap, max(BLOCKS), cap,
                                         out=o[st][l], ws=ws_a[l], stream=stream)
            bp.spec_accept(tgt[st], None, tok[st], cu_draft, 0.0, n_accepted=nacc[st], out_tokens=out[st], ws=ws_acc,
                           stream=stream)
            bp.verify_commit(ctx, nacc[st], out[st], cu_draft, cap, anchor=anchor[st], cu_kv_next=cu_kv, ws=ws_c,
                             stream=stream)

    if graph:
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            loop()
        g.replay()
    else:
        with torch.cuda.stream(stream):
            loop()
    stream.synchronize()
    for w in ws_a + [ws_acc, ws_c]:
        assert bp.get_status(w) == 0
    return dict(o=[[x.float().cpu().numpy() for x in st] for st in o], nacc=[x.cpu().numpy() for x in nacc],
                anchor=[x.cpu().numpy() for x in anchor], ctx=ctx.cpu().numpy(), cu_kv=cu_kv.cpu().numpy(),
                kc=[x.view(torch.int16).cpu().numpy().view(np.uint16) for x in kc],
                vc=[x.view(torch.int16).cpu().numpy().view(np.uint16) for x in vc],
                bt=[pl["block_table"] for pl in pools])


def oracle_loop(inp):
    S = len(BLOCKS)
    c0 = wl.offsets(CTX)
    cuq = wl.offsets(BLOCKS)
    f64 = lambda x: wl.as_f64(x, "bf16")  # noqa: E731
    K = [[list(inp["ctx_k"][l][c0[s]:c0[s + 1]]) for s in range(S)] for l in range(LAYERS)]
    Vv = [[list(inp["ctx_v"][l][c0[s]:c0[s + 1]]) for s in range(S)] for l in range(LAYERS)]
    ctx = np.array(CTX, dtype=np.int32)
    steps = []
    for st in range(STEPS):
        outs = []
        for l in range(LAYERS):
            o = np.zeros((int(cuq[-1]), HQ, D))
            for s in range(S):
                K[l][s] = K[l][s][:ctx[s]] + list(inp["kn"][st][l][cuq[s]:cuq[s + 1]])
                Vv[l][s] = Vv[l][s][:ctx[s]] + list(inp["vn"][st][l][cuq[s]:cuq[s + 1]])
                ks, vs = f64(np.array(K[l][s])), f64(np.array(Vv[l][s]))
                qs = f64(inp["q"][st][l][cuq[s]:cuq[s + 1]])
                o[cuq[s]:cuq[s + 1]], _ = oracle.block_attention(qs, ks, vs, [0, len(qs)], [0, len(ks)], HKV,
                                                                 oracle.MASK_CAUSAL)
            outs.append(o)
        acc = oracle.spec_accept(inp["target"][st], None, inp["tokens"][st], inp["cu_draft"], 0.0)
        com = oracle.verify_commit(ctx, acc["n_accepted"], acc["out_tokens"], inp["cu_draft"], inp["cap"])
        ctx = com["ctx"]
        for l in range(LAYERS):
            for s in range(S):
                K[l][s] = K[l][s][:ctx[s]]
                Vv[l][s] = Vv[l][s][:ctx[s]]
        steps.append(dict(o=outs, nacc=acc["n_accepted"], anchor=com["anchor"], cu_kv=com["cu_kv"]))
    return steps, ctx, K, Vv


def check(gpu, ref_steps, ref_ctx, K, Vv):
    cuq = wl.offsets(BLOCKS)
    S = len(BLOCKS)
    for st, r in enumerate(ref_steps):
        np.testing.assert_array_equal(gpu["nacc"][st], r["nacc"], err_msg=f"step {st}")
        np.testing.assert_array_equal(gpu["anchor"][st], r["anchor"], err_msg=f"step {st}")
        for l in range(LAYERS):
            for s in range(S):
                for h in range(HQ):
                    a = gpu["o"][st][l][cuq[s]:cuq[s + 1], h]
                    b = r["o"][l][cuq[s]:cuq[s + 1], h]
                    assert np.abs(a - b).max() <= 2e-2 * np.abs(b).max(), (st, l, s, h)
    np.testing.assert_array_equal(gpu["ctx"], ref_ctx)
    np.testing.assert_array_equal(gpu["cu_kv"], ref_steps[-1]["cu_kv"])
    for l in range(LAYERS):  # the retained rows, read through the block table
        bt = gpu["bt"][l]
        for s in range(S):
            pos = np.arange(ref_ctx[s])
            slots = bt[s, pos // PAGE] * PAGE + pos % PAGE
            np.testing.assert_array_equal(gpu["kc"][l][slots], np.array(K[l][s]))
            np.testing.assert_array_equal(gpu["vc"][l][slots], np.array(Vv[l][s]))


def test_loop_eager_and_graph_match_the_oracle():
    inp = make_inputs()
    ref_steps, ref_ctx, K, Vv = oracle_loop(inp)
    gam = np.array(BLOCKS) - 1
    rejected = sum(int((gam - r["nacc"]).sum()) for r in ref_steps)
    assert rejected > 0  # some drafts were rolled back
    for graph in (False, True):
        check(run_loop(inp, setup_device(inp), graph), ref_steps, ref_ctx, K, Vv)


def test_commit_refuses_and_changes_nothing():
    cu = to_dev(np.array([0, 3, 4], dtype=np.int32))
    out = to_dev(np.array([7, 8, 9, -1, 3, -1], dtype=np.int32))
    ctx = to_dev(np.array([10, 5], dtype=np.int32))
    ws = bp.workspace(256, dev())
    bp.verify_commit(ctx, to_dev(np.array([4, 0], dtype=np.int32)), out, cu, 100, ws=ws)  # 4 > 3 drafted
    assert bp.get_status(ws) == 6
    bp.verify_commit(ctx, to_dev(np.array([3, 1], dtype=np.int32)), out, cu, 17, ws=ws)  # next pass > 17 rows
    assert bp.get_status(ws) == 6
    np.testing.assert_array_equal(ctx.cpu().numpy(), [10, 5])


def test_commit_many_sequences():
    """More sequences than the commit CTA has threads: the chunked scan carries across chunks."""
    rng = np.random.default_rng(7)
    S = 5000
    gam = rng.integers(0, 24, size=S)
    cu = wl.offsets(gam)
    ctx = rng.integers(0, 4000, size=S).astype(np.int32)
    nacc = (rng.random(S) * (gam + 1)).astype(np.int32)
    out = rng.integers(0, 1000, size=int(cu[-1]) + S).astype(np.int32)
    ref = oracle.verify_commit(ctx, nacc, out, cu, 1 << 20)
    c = to_dev(ctx)
    anchor = torch.empty(S, dtype=torch.int32, device=dev())
    ws = bp.workspace(256, dev())
    _, cu_kv = bp.verify_commit(c, to_dev(nacc), to_dev(out), to_dev(cu), 1 << 20, anchor=anchor, ws=ws)
    assert bp.get_status(ws) == 0
    np.testing.assert_array_equal(c.cpu().numpy(), ref["ctx"])
    np.testing.assert_array_equal(anchor.cpu().numpy(), ref["anchor"])
    np.testing.assert_array_equal(cu_kv.cpu().numpy(), ref["cu_kv"])
