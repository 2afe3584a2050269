"""The kernels' wind-down path, taken on purpose on the GPU.

Every device-side wait of the library is bounded.  When a wait for work to arrive expires, the kernel
records BP_ERR_TIMEOUT in the workspace error word, waits out its own copies and tensor-core operations
still in flight (a separate drain budget), releases its tensor memory and returns, so the context stays
usable.  A test-only build of the library (libblockpilot_shortwait.so, compiled with
BP_TEST_SHORT_WAITS) turns every such wait into a single non-blocking test, which finds the data of a
copy just issued still in flight: the attention kernel (both key splits), the cluster acceptance
kernel (T = 1 and T = 0) and the verify epilogue's streamed LM head (T = 1 and T = 0) then take that
path.  Nothing faults and nothing waits on an event that never
comes: the drains wait for copies the kernel itself issued.

The test build runs in a child process, which also checks that its CUDA context still works after
the expired waits.  The parent then runs the product library on fresh workspaces over the same inputs
and compares with the oracle.
"""
import json
import os
import subprocess
import sys

import pytest
import torch

import paper_2606_31315_gb300 as bp
from paper_2606_31315_gb300 import _build
from paper_2606_31315_gb300 import workloads as wl

from _gpu import ATTN_TOL, LSE_TOL, attention_errors, compare_accept, run_attention

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import json, os, sys
sys.path.insert(0, sys.argv[1])
import numpy as np, torch
from paper_2606_31315_gb300 import _build
_build.LIB = _build.TEST_LIB            # the short-wait build only
import paper_2606_31315_gb300 as bp
from paper_2606_31315_gb300 import workloads as wl
dev = torch.device("cuda:0")
bf = lambda x: torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).to(dev).view(torch.bfloat16)
t = lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(dev)
out = {}
a = wl.attention_inputs(wl.get("qwen3_4b"))
for split in ("cluster", "flat"):
    os.environ["BP_ATTENTION_SPLIT"] = split
    ws = bp.workspace(bp.block_attention_workspace_size(1, 16, 32, 8, 128), dev)
    bp.block_attention(bf(a["q"]), bf(a["k"]), bf(a["v"]), t(a["cu_q"]), t(a["cu_kv"]), a["max_q_len"],
                       a["max_kv_len"], ws=ws)
    out["attention_" + split] = bp.get_status(ws)
w = wl.get("qwen3_4b")  # one sequence: the bonus row's copy is waited for right after it is issued
for temp in (1.0, 0.0):
    inp = wl.accept_inputs(w, temp)
    ws = bp.workspace(bp.spec_accept_workspace_size(1, 15, w.vocab), dev)
    bp.spec_accept(t(inp["target_logits"]), t(inp["draft_logits"]) if temp > 0 else None, t(inp["draft_tokens"]),
                   t(inp["cu_draft"]), temp, t(inp["u_accept"]), t(inp["u_sample"]), ws=ws)
    out["accept_t%d" % temp] = bp.get_status(ws)
# the verify epilogue's streamed path (more than 64 rows): two 128-row halves at T = 1, one at T = 0
w5 = wl.custom(seed=41, ctx=(0,) * 5, block=(16,) * 5, vocab=30000)
for temp in (1.0, 0.0):
    inp = wl.lm_head_inputs(w5, temp, hidden=128)
    ws = bp.workspace(bp.verify_epilogue_workspace_size(5, len(inp["draft_tokens"]), inp["vocab"]), dev)
    bp.verify_epilogue(bf(inp["w"]), bf(inp["h_target"]), bf(inp["h_draft"]) if temp > 0 else None,
                       t(inp["draft_tokens"]), t(inp["cu_draft"]), temp, t(inp["u_accept"]), t(inp["u_sample"]),
                       ws=ws)
    out["verify_stream_t%d" % temp] = bp.get_status(ws)
x = torch.arange(1 << 20, device=dev, dtype=torch.float32)  # the context still runs work
out["context_ok"] = bool(float(x.sum().item()) == float((1 << 20) * ((1 << 20) - 1) // 2))
print(json.dumps(out))
"""


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    bp.build()
    bp.load()


def test_expired_waits_report_timeout_and_leave_the_context_usable():
    assert os.path.exists(_build.TEST_LIB), "the short-wait test build is made by build()"
    res = subprocess.run([sys.executable, "-c", CHILD, ROOT], capture_output=True, text=True, timeout=600,
                         env={k: v for k, v in os.environ.items() if k != "BP_ATTENTION_SPLIT"})
    assert res.returncode == 0, res.stderr[-3000:]
    got = json.loads([ln for ln in res.stdout.splitlines() if ln.startswith("{")][-1])
    timeout = 5  # BP_ERR_TIMEOUT
    assert got == {"attention_cluster": timeout, "attention_flat": timeout, "accept_t1": timeout, "accept_t0": timeout,
                   "verify_stream_t1": timeout, "verify_stream_t0": timeout, "context_ok": True}, got


def test_product_library_after_the_timeouts():
    """The same inputs through the product library on fresh workspaces: the oracle's results."""
    a = wl.attention_inputs(wl.get("qwen3_4b"))
    for split in ("cluster", "flat"):
        o, lse = run_attention(a, bp.MASK_CAUSAL, split)
        err, lerr = attention_errors(o, lse, a, bp.MASK_CAUSAL, [0])
        assert err <= ATTN_TOL and lerr <= LSE_TOL
    for temp in (1.0, 0.0):
        compare_accept(wl.accept_inputs(wl.get("qwen3_4b"), temp), temp)
    from test_gpu_verify_epilogue import compare, run_gpu, run_oracle

    w5 = wl.custom(seed=41, ctx=(0,) * 5, block=(16,) * 5, vocab=30000)
    for temp in (1.0, 0.0):
        inp = wl.lm_head_inputs(w5, temp, hidden=128)
        compare(inp, temp, run_gpu(inp, temp, want_logits=True), run_oracle(inp, temp))
