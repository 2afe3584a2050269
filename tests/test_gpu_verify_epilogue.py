"""GPU parity of bp_verify_epilogue (LM head fused with the lossless acceptance) against the fp64
oracle (oracle.verify_epilogue: fp64 logits of the same bf16 operands, then the acceptance).

Tolerances, derived from the arithmetic.  A bf16 x bf16 product is exact in fp32, so a logit differs
from the fp64 value only by the fp32 accumulation of H products; with a rounding error of at most
2^-24 of the running sum per addition and errors that do not conspire, |l - l_ref| <= eps =
8 sqrt(H) 2^-24 sum_k |w_k h_k| (a probabilistic bound: exceeded with probability below 1e-14 per
logit).  A ratio a = min(1, p(x)/q(x)) then moves by at most about 4 eps / T (two logits, two
log-normalisers) and a cumulative mass of the draw distribution by at most 4 eps / T, so:
  - logits_out within eps of the oracle element by element;
  - accept_prob within 4.1 eps_max / T + 2e-6;
  - n_accepted and out_tokens bit-exact for every sequence whose ratio tests and draw are not
    within those margins of a decision boundary (the oracle's ratio_margin / cdf_margin); flagged
    sequences must follow from the GPU's own accept_prob and emit a token of the near-tie set;
  - T = 0: bit-exact unless a target row's top-two logits are within 2 eps (then the GPU's argmax
    must be one of the near-maximal entries).
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2606_31315_gb300 as bp
from paper_2606_31315_gb300 import workloads as wl

from _gpu import dev, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    bp.build()
    bp.load()


def eps_of(mag: np.ndarray, hidden: int) -> np.ndarray:
    return 8.0 * np.sqrt(hidden) * 2.0 ** -24 * mag


def run_gpu(inp: dict, temperature: float, u_accept=None, u_sample=None, want_logits=False, ws=None, dev_inp=None):
    d = dev_inp or device_inputs(inp, temperature)
    ua = to_dev(inp["u_accept"] if u_accept is None else u_accept)
    us = to_dev(inp["u_sample"] if u_sample is None else u_sample)
    rows = d["h_target"].shape[0] + (d["h_draft"].shape[0] if d["h_draft"] is not None else 0)
    logits = torch.full((rows, inp["vocab"]), float("nan"), device=dev()) if want_logits else None
    if ws is None:
        ws = bp.workspace(bp.verify_epilogue_workspace_size(len(inp["cu_draft"]) - 1, len(inp["draft_tokens"]),
                                                      inp["vocab"]), dev())
    n_acc, out, ap = bp.verify_epilogue(d["w"], d["h_target"], d["h_draft"], d["tokens"], d["cu"], temperature, ua, us,
                                        logits_out=logits, ws=ws)
    status = bp.get_status(ws)
    return (n_acc.cpu().numpy(), out.cpu().numpy(), ap.cpu().numpy(), status,
            None if logits is None else logits.cpu().numpy())


def device_inputs(inp: dict, temperature: float) -> dict:
    return dict(w=to_dev(inp["w"], "bf16"), h_target=to_dev(inp["h_target"], "bf16"),
                h_draft=to_dev(inp["h_draft"], "bf16") if temperature > 0 else None,
                tokens=to_dev(inp["draft_tokens"]), cu=to_dev(inp["cu_draft"]))


def run_oracle(inp: dict, temperature: float):
    return oracle.verify_epilogue(inp["w"], inp["h_target"], inp["h_draft"] if temperature > 0 else None,
                                  inp["draft_tokens"], inp["cu_draft"], temperature, inp["u_accept"], inp["u_sample"],
                                  with_abs=True)


def _draw_weights(ref: dict, s: int, k: int, temperature: float, cu) -> np.ndarray:
    from scipy import special

    gamma = cu[s + 1] - cu[s]
    p = special.softmax(ref["target_logits"][cu[s] + s + k] / temperature)
    if k < gamma:
        r = np.maximum(p - special.softmax(ref["draft_logits"][cu[s] + k] / temperature), 0.0)
        if r.sum() > 0:
            return r
    return p


def compare(inp: dict, temperature: float, gpu, ref, check_logits: bool = True):
    """Asserts parity under the derived tolerances; returns (flagged sequences, sequences)."""
    n_acc, out, ap, status, logits = gpu
    assert status == 0, f"device error status {status}"
    H = inp["hidden"]
    cu = inp["cu_draft"]
    S = len(cu) - 1
    td = int(cu[-1])
    eps_t = eps_of(ref["target_abs"], H)
    if check_logits and logits is not None:
        err = np.abs(logits[:td + S] - ref["target_logits"])
        assert np.all(err <= eps_t), (err.max(), (err / eps_t).max())
        if temperature > 0 and td:
            eps_d = eps_of(ref["draft_abs"], H)
            errd = np.abs(logits[td + S:] - ref["draft_logits"])
            assert np.all(errd <= eps_d), (errd.max(), (errd / eps_d).max())
    flagged = 0
    if temperature == 0:
        tl = ref["target_logits"]
        for s in range(S):
            lo, hi = cu[s] + s, cu[s + 1] + s + 1
            rows = tl[lo:hi]
            top2 = np.sort(rows, axis=1)[:, -2:]
            near = (top2[:, 1] - top2[:, 0]) < 2 * eps_t[lo:hi].max(axis=1)
            k = int(n_acc[s])
            if not near.any():
                assert k == ref["n_accepted"][s], (s, k, ref["n_accepted"][s])
                np.testing.assert_array_equal(out[lo:hi], ref["out_tokens"][lo:hi], err_msg=f"sequence {s}")
                np.testing.assert_array_equal(ap[cu[s]:cu[s + 1]], ref["accept_prob"][cu[s]:cu[s + 1]])
                continue
            flagged += 1
            # valid: the emitted tokens are near-maximal entries of their rows, the prefix follows
            for j in range(k + 1):
                tok = out[lo + j]
                assert rows[j, tok] >= rows[j].max() - 2 * eps_t[lo + j].max(), (s, j)
            np.testing.assert_array_equal(out[lo:lo + k], inp["draft_tokens"][cu[s]:cu[s] + k])
            assert np.all(out[lo + k + 1:hi] == -1)
        return flagged, S
    eps_max = float(eps_t.max())
    if td:
        eps_max = max(eps_max, float(eps_of(ref["draft_abs"], H).max()))
    d_a = 4.1 * eps_max / temperature + 2e-6
    d_c = 4.1 * eps_max / temperature + 1e-5
    assert np.abs(ap - ref["accept_prob"]).max(initial=0.0) <= d_a, np.abs(ap - ref["accept_prob"]).max()
    flags = (ref["ratio_margin"] < d_a) | (ref["cdf_margin"] < d_c)
    for s in range(S):
        lo, hi = cu[s] + s, cu[s + 1] + s + 1
        gamma = cu[s + 1] - cu[s]
        k = int(n_acc[s])
        ua = inp["u_accept"][cu[s]:cu[s + 1]]
        rej = np.nonzero(~(ua < ap[cu[s]:cu[s + 1]]))[0]
        assert k == (rej[0] if len(rej) else gamma), (s, k, rej)  # the prefix follows from its own a_i
        if not flags[s]:
            assert k == ref["n_accepted"][s], (s, k, ref["n_accepted"][s])
            np.testing.assert_array_equal(out[lo:hi], ref["out_tokens"][lo:hi], err_msg=f"sequence {s}")
            continue
        flagged += 1
        kr = int(ref["n_accepted"][s])
        if k != kr:
            j = min(k, kr)
            assert abs(float(ua[j]) - ref["accept_prob"][cu[s] + j]) < d_a, (s, k, kr)
        np.testing.assert_array_equal(out[lo:lo + k], inp["draft_tokens"][cu[s]:cu[s] + k])
        assert np.all(out[lo + k + 1:hi] == -1)
        w = _draw_weights(ref, s, k, temperature, cu)
        c = np.cumsum(w)
        thr = float(inp["u_sample"][s]) * c[-1]
        prev = np.concatenate([[0.0], c[:-1]])
        ok = np.nonzero((w > 0) & (prev - d_c <= thr) & (thr < c + d_c))[0]
        assert out[lo + k] in ok, (s, k, out[lo + k])
    return flagged, S


CASES = [
    # (seed, blocks, vocab, hidden)
    (11, (8,), 1000, 64),
    (12, (16, 1, 5), 5003, 128),
    (13, (4, 4, 4, 4), 20000, 256),
    (14, (1,), 777, 64),
]


@pytest.mark.parametrize("temp", [1.0, 0.0])
@pytest.mark.parametrize("case", CASES)
def test_small_cases_and_logits(case, temp):
    seed, blocks, vocab, hidden = case
    w = wl.custom(seed=seed, ctx=(0,) * len(blocks), block=blocks, vocab=vocab)
    inp = wl.lm_head_inputs(w, temp, hidden=hidden)
    compare(inp, temp, run_gpu(inp, temp, want_logits=True), run_oracle(inp, temp))


@pytest.mark.parametrize("temp", [1.0, 0.0])
def test_sixty_four_rows(temp):
    """rows = 2 * 30 drafts + 4 sequences = 64 at T > 0 (64 TMEM columns per tile)."""
    w = wl.custom(seed=21, ctx=(0,) * 4, block=(16, 9, 1, 8), vocab=30011)
    inp = wl.lm_head_inputs(w, temp, hidden=192)
    compare(inp, temp, run_gpu(inp, temp, want_logits=True), run_oracle(inp, temp))


def test_sixteen_tiles_per_cta():
    """A vocabulary of 300,000: 16 tiles of 128 entries per CTA on 152 SMs (512 TMEM columns)."""
    w = wl.custom(seed=22, ctx=(0,) * 2, block=(8, 8), vocab=300000)
    inp = wl.lm_head_inputs(w, 1.0, hidden=64)
    compare(inp, 1.0, run_gpu(inp, 1.0, want_logits=True), run_oracle(inp, 1.0))


def test_drafter_equal_to_target_accepts_everything():
    """Drafter states equal to the target's: q = p, so every draft is accepted and the bonus token is
    drawn from p_gamma.  The two rows sit at different MMA columns, whose fp32 accumulation order may
    differ in the last bit, so a_i is 1 to within a few ulps rather than exactly."""
    w = wl.custom(seed=23, ctx=(0,) * 3, block=(16, 4, 9), vocab=151936)
    inp = wl.lm_head_inputs(w, 1.0, hidden=256)
    cu = inp["cu_draft"]
    trow = np.concatenate([np.arange(cu[s], cu[s + 1]) + s for s in range(3)])
    inp["h_draft"] = inp["h_target"][trow]
    gpu = run_gpu(inp, 1.0)
    np.testing.assert_array_equal(gpu[0], np.diff(cu))
    assert np.all(np.abs(gpu[2] - 1.0) <= 4 * 2.0 ** -24), gpu[2]
    compare(inp, 1.0, gpu, run_oracle(inp, 1.0))


@pytest.fixture(scope="module")
def qwen_weight():
    w = wl.get("qwen3_4b")
    return wl.lm_head_weight(w.vocab, wl.LM_HIDDEN["qwen3_4b"], w.logit_std, w.seed)


def planted_uniforms(inp: dict, ref: dict, temperature: float, rng):
    """Uniforms chosen from the oracle so that every decision has a wide margin: accepted drafts get
    u_i = a_i / 2 (a_i >= 0.2), the rejected one u_j = (1 + a_j) / 2 (a_j <= 0.8), and u_s lands in
    the middle of the interval of a token of unnormalised draw mass >= 0.08.  Returns
    (u_accept, u_sample, planted) -- planted[s] False where no such token exists.  The draw's
    margin is half the token's unnormalised mass (>= 0.08), far above the derived tolerance."""
    cu = inp["cu_draft"]
    S = len(cu) - 1
    a = ref["accept_prob"]
    ua = np.zeros(int(cu[-1]), dtype=np.float32)
    us = np.zeros(S, dtype=np.float32)
    planted = np.zeros(S, dtype=bool)
    for s in range(S):
        g = int(cu[s + 1] - cu[s])
        aa = a[cu[s]:cu[s + 1]]
        stop = next((i for i in range(g) if aa[i] < 0.2), g)  # cannot be accepted with a margin
        choices = [j for j in range(stop + 1) if j == g or aa[j] <= 0.8]
        j, big, w = int(rng.choice(choices)), [], None
        for cand in rng.permutation(choices):  # a first rejection whose draw has a token of large mass
            wc = _draw_weights(ref, s, int(cand), temperature, cu)  # unnormalised: margins are in these units
            if (wc >= 0.08).any():
                j, w, big = int(cand), wc, np.nonzero(wc >= 0.08)[0]
                break
        for i in range(g):
            ua[cu[s] + i] = aa[i] / 2 if i < j else ((1 + aa[i]) / 2 if i == j else float(rng.random()))
        if len(big):
            t = int(rng.choice(big))
            us[s] = (w[:t].sum() + w[t] / 2) / w.sum()
            planted[s] = True
        else:
            us[s] = float(rng.random())
    return ua, us, planted


@pytest.mark.parametrize("temp", [1.0, 0.0])
def test_qwen3_4b_full(qwen_weight, temp):
    """The full Qwen3-4B LM head (151936 x 2560 bf16, 778 MB) on the batch-1 verify step, launched as
    the benchmark launches it.  At T = 1 also twelve draws with planted uniforms (every decision far
    from its boundary) over confident target rows, which must match the oracle exactly."""
    w = wl.get("qwen3_4b")
    inp = wl.lm_head_inputs(w, temp, weight=qwen_weight)
    ref = run_oracle(inp, temp)
    d = device_inputs(inp, temp)
    ws = bp.workspace(bp.verify_epilogue_workspace_size(1, len(inp["draft_tokens"]), inp["vocab"]), dev())
    compare(inp, temp, run_gpu(inp, temp, want_logits=True, ws=ws, dev_inp=d), ref)
    if temp == 0:
        return
    # confident target rows (a dominant token in every row not pushed toward its draft), so that
    # the draws have tokens of large mass to plant the sampling uniform in; four input sets (the
    # first rejection falls at different positions), three draws each
    exact, ks = 0, set()
    for seed in range(4):
        ws_in = wl.custom(seed=100 + seed, ctx=w.ctx, block=w.block, vocab=w.vocab, logit_std=w.logit_std)
        inp = wl.lm_head_inputs(ws_in, temp, hidden=wl.LM_HIDDEN["qwen3_4b"], weight=qwen_weight, target_peak=22.0)
        ref = run_oracle(inp, temp)
        d = device_inputs(inp, temp)
        rng = np.random.default_rng(seed)
        for _ in range(3):
            ua, us, planted = planted_uniforms(inp, ref, temp, rng)
            trial_inp = dict(inp, u_accept=ua, u_sample=us)
            tref = dict(ref)
            tref.update(oracle.spec_accept(ref["target_logits"], ref["draft_logits"], inp["draft_tokens"],
                                           inp["cu_draft"], temp, ua, us))
            flagged, _ = compare(trial_inp, temp, run_gpu(trial_inp, temp, ws=ws, dev_inp=d), tref,
                                 check_logits=False)
            if planted.all():
                assert flagged == 0  # every margin is far above the derived tolerance: bit-exact
                exact += 1
                ks.add(int(tref["n_accepted"][0]))
    assert exact >= 8 and len(ks) >= 2, (exact, ks)


def test_workspace_reuse_is_deterministic():
    """Repeated calls on one workspace give identical results (the grid-barrier counters return to
    zero after every call)."""
    w = wl.custom(seed=24, ctx=(0,) * 2, block=(12, 6), vocab=70000)
    inp = wl.lm_head_inputs(w, 1.0, hidden=128)
    d = device_inputs(inp, 1.0)
    ws = bp.workspace(bp.verify_epilogue_workspace_size(2, len(inp["draft_tokens"]), inp["vocab"]), dev())
    first = run_gpu(inp, 1.0, ws=ws, dev_inp=d)
    for _ in range(3):
        again = run_gpu(inp, 1.0, ws=ws, dev_inp=d)
        for a, b in zip(first[:3], again[:3]):
            np.testing.assert_array_equal(a, b)
    assert ws[256:264].view(torch.int32).cpu().tolist() == [0, 0]


def test_out_of_range_draft_token_sets_the_device_flag():
    w = wl.custom(seed=25, ctx=(0,), block=(6,), vocab=4000)
    inp = wl.lm_head_inputs(w, 1.0, hidden=64)
    inp["draft_tokens"] = inp["draft_tokens"].copy()
    inp["draft_tokens"][2] = 4000
    gpu = run_gpu(inp, 1.0)
    assert gpu[3] == 6  # BP_ERR_DEVICE_FLAG


def test_host_rejects_unsupported_shapes():
    w = wl.custom(seed=26, ctx=(0,) * 3, block=(16, 16, 16), vocab=1000)
    inp = wl.lm_head_inputs(w, 1.0, hidden=64)
    inp["w"] = np.ascontiguousarray(np.concatenate([inp["w"], inp["w"][:, :32]], axis=1))  # hidden 96
    inp["h_target"] = np.ascontiguousarray(np.concatenate([inp["h_target"], inp["h_target"][:, :32]], axis=1))
    inp["h_draft"] = np.ascontiguousarray(np.concatenate([inp["h_draft"], inp["h_draft"][:, :32]], axis=1))
    with pytest.raises(bp.BlockPilotError):
        run_gpu(inp, 1.0)


# ---- more than 64 rows: the LM head streamed through tensor memory, statistics formed in its epilogue
STREAM_CASES = [
    # (seed, blocks, vocab, hidden): rows at T > 0 / T = 0.  Logits leave by TMA stores where a group's
    # rows are contiguous and rows are 16-byte aligned, else by whole-line stores
    (31, (16, 16, 16), 1000, 64),              # 93 / 48: one 128-row half; T = 0 resident
    (32, (16,) * 5, 30011, 128),               # 155 / 80: two halves; odd vocabulary (4-byte stores)
    (33, (16,) * 10, 20000, 192),              # 310 / 160: two groups of rows at T > 0
    (34, (16,) * 9 + (5,), 12344, 64),         # 288 / 149: target rows end off an 8-row boundary (16-byte
                                               # stores in the first group)
    (35, (1,) * 70, 4096, 64),                 # 70 / 70: blocks of one position (bonus draws only)
]


@pytest.mark.parametrize("temp", [1.0, 0.0])
@pytest.mark.parametrize("case", STREAM_CASES)
def test_streamed_rows(case, temp):
    seed, blocks, vocab, hidden = case
    w = wl.custom(seed=seed, ctx=(0,) * len(blocks), block=blocks, vocab=vocab)
    inp = wl.lm_head_inputs(w, temp, hidden=hidden)
    ref = run_oracle(inp, temp)
    compare(inp, temp, run_gpu(inp, temp, want_logits=True), ref)
    compare(inp, temp, run_gpu(inp, temp), ref, check_logits=False)  # logits only where the path needs them


@pytest.mark.parametrize("temp", [1.0, 0.0])
def test_streamed_ragged_batch_rows(temp):
    """The ragged 32-request batch's blocks (8 to 24 positions: 502 target rows and at T = 1 470
    drafter rows, 972 rows in four groups of the streamed projection), over a 32000-entry vocabulary."""
    rg = wl.get("ragged")
    w = wl.custom(seed=38, ctx=(0,) * rg.num_seqs, block=rg.block, vocab=32000, logit_std=rg.logit_std)
    inp = wl.lm_head_inputs(w, temp, hidden=256)
    ref = run_oracle(inp, temp)
    compare(inp, temp, run_gpu(inp, temp, want_logits=True), ref)
    compare(inp, temp, run_gpu(inp, temp), ref, check_logits=False)


def test_streamed_workspace_reuse_is_deterministic():
    """Repeated streamed calls on one workspace give identical results (the draw's tickets return to
    zero, the slice statistics are merged in a fixed order)."""
    w = wl.custom(seed=36, ctx=(0,) * 6, block=(16, 12, 16, 3, 16, 9), vocab=50000)
    inp = wl.lm_head_inputs(w, 1.0, hidden=128)
    d = device_inputs(inp, 1.0)
    ws = bp.workspace(bp.verify_epilogue_workspace_size(6, len(inp["draft_tokens"]), inp["vocab"]), dev())
    first = run_gpu(inp, 1.0, ws=ws, dev_inp=d)
    for _ in range(3):
        again = run_gpu(inp, 1.0, ws=ws, dev_inp=d)
        for a, b in zip(first[:3], again[:3]):
            np.testing.assert_array_equal(a, b)


def test_streamed_out_of_range_draft_token_sets_the_device_flag():
    w = wl.custom(seed=37, ctx=(0,) * 5, block=(16,) * 5, vocab=4000)
    inp = wl.lm_head_inputs(w, 1.0, hidden=64)
    inp["draft_tokens"] = inp["draft_tokens"].copy()
    inp["draft_tokens"][7] = -3
    gpu = run_gpu(inp, 1.0)
    assert gpu[3] == 6  # BP_ERR_DEVICE_FLAG


@pytest.mark.parametrize("temp", [1.0, 0.0])
def test_long_context_batch_full_head(qwen_weight, temp):
    """The long-context verify batch (8 sequences x 16 positions: 128 target rows and, at T = 1, 120
    drafter rows -- 248 rows) through the full Qwen3-4B LM head (151936 x 2560), as the benchmark
    launches it.  At T = 1 also draws with planted uniforms over confident target rows, which must
    match the oracle exactly."""
    lc = wl.get("long_context")
    base = wl.custom(seed=lc.seed, ctx=(0,) * lc.num_seqs, block=lc.block, vocab=lc.vocab, logit_std=lc.logit_std)
    inp = wl.lm_head_inputs(base, temp, hidden=wl.LM_HIDDEN["long_context"], weight=qwen_weight)
    ref = run_oracle(inp, temp)
    d = device_inputs(inp, temp)
    ws = bp.workspace(bp.verify_epilogue_workspace_size(lc.num_seqs, len(inp["draft_tokens"]), inp["vocab"]), dev())
    compare(inp, temp, run_gpu(inp, temp, want_logits=True, ws=ws, dev_inp=d), ref)
    compare(inp, temp, run_gpu(inp, temp, ws=ws, dev_inp=d), ref, check_logits=False)
    if temp == 0:
        return
    exact, ks = 0, set()
    for seed in range(2):
        ws_in = wl.custom(seed=200 + seed, ctx=(0,) * lc.num_seqs, block=lc.block, vocab=lc.vocab,
                          logit_std=lc.logit_std)
        inp = wl.lm_head_inputs(ws_in, temp, hidden=wl.LM_HIDDEN["long_context"], weight=qwen_weight,
                                target_peak=22.0)
        ref = run_oracle(inp, temp)
        d = device_inputs(inp, temp)
        rng = np.random.default_rng(seed)
        for _ in range(2):
            ua, us, planted = planted_uniforms(inp, ref, temp, rng)
            trial_inp = dict(inp, u_accept=ua, u_sample=us)
            tref = dict(ref)
            tref.update(oracle.spec_accept(ref["target_logits"], ref["draft_logits"], inp["draft_tokens"],
                                           inp["cu_draft"], temp, ua, us))
            flagged, _ = compare(trial_inp, temp, run_gpu(trial_inp, temp, ws=ws, dev_inp=d), tref,
                                 check_logits=False)
            if planted.all():
                assert flagged == 0  # every margin is far above the derived tolerance: bit-exact
            # a planted sequence's margins (>= 0.04) are far above the tolerance: compared bit-exactly
            exact += int(planted.sum())
            ks.update(int(k) for k, pl in zip(tref["n_accepted"], planted) if pl)
    assert exact >= 24 and len(ks) >= 3, (exact, ks)
