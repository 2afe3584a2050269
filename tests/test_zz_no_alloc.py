"""bp_spec_accept_noalloc: the acceptance step for callers that cannot allocate device memory.

Some callers have no way to provide a workspace: a plugin running inside another inference
engine that only receives its input and output buffers, or a serving loop that must not call
cudaMalloc while requests are in flight (cudaMalloc can synchronize the device).  This entry
point keeps its scratch in a fixed array inside the library instead.  The test calls it through
the C ABI twice in a row, on two different problems (so the second call runs on whatever the
first left in the shared array), and checks each result against bp_spec_accept with a
caller-provided workspace: emitted tokens and accepted lengths identical, acceptance
probabilities within 1e-5.  It also checks that a problem too large for the array is refused, and
which kernels run: the throughput kernels when their regions fit in the array, else the single one.
"""
import ctypes

import numpy as np
import pytest
import torch

import paper_2606_31315_gb300 as bp
from paper_2606_31315_gb300 import workloads as wl

from _gpu import compare_accept, run_oracle_accept

pytestmark = pytest.mark.gpu

PROB_TOL = 1e-5


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    bp.build()
    lib = bp.load()
    vp, i32, f32 = ctypes.c_void_p, ctypes.c_int, ctypes.c_float
    lib.bp_spec_accept_noalloc.argtypes = [vp, vp, vp, vp, i32, i32, i32, f32, vp, vp, vp, vp, vp, vp, vp]
    lib.bp_spec_accept_noalloc.restype = i32
    return lib


def _p(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _inputs(name, temp):
    inp = wl.accept_inputs(wl.get(name), temp)
    g = {k: torch.from_numpy(np.ascontiguousarray(inp[k])).cuda() for k in
         ("target_logits", "draft_logits", "draft_tokens", "cu_draft", "u_accept", "u_sample")}
    if temp == 0:
        g["draft_logits"] = None
    return g


def _noalloc(lib, g, temp):
    s = g["cu_draft"].numel() - 1
    td = g["draft_tokens"].numel()
    vocab = g["target_logits"].shape[1]
    n_acc = torch.full((s,), -7, dtype=torch.int32, device="cuda")
    out = torch.full((td + s,), -7, dtype=torch.int32, device="cuda")
    ap = torch.full((td,), -1.0, dtype=torch.float32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    stream = torch.cuda.current_stream()
    rc = lib.bp_spec_accept_noalloc(_p(g["target_logits"]), _p(g["draft_logits"]), _p(g["draft_tokens"]),
                                    _p(g["cu_draft"]), s, td, vocab, float(temp), _p(g["u_accept"]),
                                    _p(g["u_sample"]), _p(n_acc), _p(out), _p(ap), _p(err),
                                    ctypes.c_void_p(stream.cuda_stream))
    assert rc == 0, lib.bp_error_string(rc)
    torch.cuda.synchronize()
    assert err.item() == 0
    return n_acc.cpu().numpy(), out.cpu().numpy(), ap.cpu().numpy()


def _kernels(fn):
    """Names of the GPU kernels fn() launches (a warm-up session first: the first may miss some)."""
    from torch.profiler import ProfilerActivity, profile

    for _ in range(2):
        with profile(activities=[ProfilerActivity.CUDA]) as prof:
            fn()
            torch.cuda.synchronize()
    return {e.name for e in prof.events() if "bp::" in e.name}


def _with_workspace(g, temp):
    n_acc, out, ap = bp.spec_accept(g["target_logits"], g["draft_logits"], g["draft_tokens"], g["cu_draft"], temp,
                                    g["u_accept"], g["u_sample"])
    return n_acc.cpu().numpy(), out.cpu().numpy(), ap.cpu().numpy()


def _same(a, b):
    np.testing.assert_array_equal(a[0], b[0])
    np.testing.assert_array_equal(a[1], b[1])
    assert np.abs(a[2] - b[2]).max() <= PROB_TOL


@pytest.mark.parametrize("temp", [1.0, 0.0])
def test_two_calls_in_a_row_match_the_workspace_entry_point(lib, temp):
    first = _inputs("ragged", 1.0)        # 32 sequences, 502 target rows
    second = _inputs("qwen3_4b", temp)    # 1 sequence, 16 target rows
    _same(_noalloc(lib, first, 1.0), _with_workspace(first, 1.0))
    _same(_noalloc(lib, second, temp), _with_workspace(second, temp))


def test_the_array_holds_the_throughput_kernels_when_they_fit(lib):
    """The ragged batch's throughput-kernel regions (under 1 MB) fit the fixed array: those kernels run."""
    g = _inputs("ragged", 1.0)
    names = _kernels(lambda: _noalloc(lib, g, 1.0))
    assert any("batch_stats_kernel" in n for n in names) and any("batch_draw_kernel" in n for n in names), names
    assert not any("accept_kernel" in n for n in names), names


def test_too_large_problem_is_refused(lib):
    # 4M single-token sequences: the per-sequence counters alone need 16 MB, more than the fixed
    # array holds, so the call must be refused before anything is launched.  Every buffer is real
    # and sized for the problem, so the call is safe even if it were (wrongly) launched.
    s, vocab = 4_000_000, 16
    target = torch.zeros((s, vocab), dtype=torch.float32, device="cuda")
    cu = torch.zeros(s + 1, dtype=torch.int32, device="cuda")
    u = torch.zeros(s, dtype=torch.float32, device="cuda")
    n_acc = torch.zeros(s, dtype=torch.int32, device="cuda")
    out = torch.zeros(s, dtype=torch.int32, device="cuda")
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    rc = lib.bp_spec_accept_noalloc(_p(target), None, None, _p(cu), s, 0, vocab, 1.0, None, _p(u), _p(n_acc),
                                    _p(out), None, None, stream)
    torch.cuda.synchronize()
    assert rc == 4  # BP_ERR_WORKSPACE


def test_large_batch_falls_back_to_the_single_kernel(lib):
    # 200000 sequences of one draft each over a 16-token vocabulary: 400000 target rows.  The
    # single kernel's scratch (tickets, ratios, row tokens: about 3.2 MB) fits in the fixed array;
    # the throughput kernels' regions on top of it (chunk statistics of 600000 rows, per-sequence
    # draw masses: about 15 MB more) do not, so the call runs the single kernel (checked by the
    # kernels it launches).  Checked against the oracle on the first 20000 sequences.
    s, v = 200_000, 16
    rng = np.random.default_rng(81)
    tl = rng.normal(0.0, 2.0, size=(2 * s, v)).astype(np.float32)
    dl = rng.normal(0.0, 2.0, size=(s, v)).astype(np.float32)
    inp = dict(target_logits=tl, draft_logits=dl, draft_tokens=rng.integers(0, v, size=s).astype(np.int32),
               cu_draft=np.arange(s + 1, dtype=np.int32), u_accept=rng.random(s, dtype=np.float32),
               u_sample=rng.random(s, dtype=np.float32))
    assert bp.spec_accept_workspace_size(s, s, v) > (8 << 20)  # the throughput kernels' layout is larger
    g = {k: torch.from_numpy(np.ascontiguousarray(x)).cuda() for k, x in inp.items()}
    names = _kernels(lambda: _noalloc(lib, g, 1.0))
    assert any("accept_kernel" in n for n in names) and not any("batch_" in n for n in names), names
    n_acc, out, ap = _noalloc(lib, g, 1.0)
    m = 20_000
    small = {k: x[: 2 * m] if k == "target_logits" else x[: m + 1] if k == "cu_draft" else x[:m]
             for k, x in inp.items()}
    compare_accept(small, 1.0, gpu=(n_acc[:m], out[: 2 * m], ap[:m], 0), ref=run_oracle_accept(small, 1.0))
