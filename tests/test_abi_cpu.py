"""Host-side checks of the C-ABI library (no GPU needed): it builds for sm_103a, loads,
exports exactly the symbols include/blockpilot.h declares, validates arguments on the host
before touching CUDA, and has no CPU fallback.  Also checks that the product package never
reaches the oracle."""
import ast
import ctypes
import os
import re

import pytest

import paper_2606_31315_gb300 as bp
from paper_2606_31315_gb300 import _build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "blockpilot.h")


@pytest.fixture(scope="module")
def lib():
    _build.build()
    return bp.load()


def _declared():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"BP_API\s+[\w\s\*]*?\b(bp_\w+)\s*\(", text)))


def _exported():
    import subprocess

    out = subprocess.run(["nm", "-D", "--defined-only", _build.LIB], capture_output=True, text=True, check=True).stdout
    return sorted({line.split()[-1] for line in out.splitlines() if " T " in line and line.split()[-1].startswith("bp_")})


def test_exports_match_header(lib):
    declared = _declared()
    assert len(declared) >= 9
    assert _exported() == declared
    for name in declared:
        assert hasattr(lib, name)


def test_version_and_error_strings(lib):
    assert lib.bp_abi_version() == 3
    for code in range(7):
        assert lib.bp_error_string(code).startswith(b"BP_")
    assert lib.bp_error_string(99) == b"unknown bp_status"


def test_workspace_sizes(lib):
    assert bp.block_attention_workspace_size(1, 16, 32, 8, 128) >= 256
    w = bp.spec_accept_workspace_size(1, 15, 151936)
    assert w > 256 and w % 256 == 0
    assert bp.spec_accept_workspace_size(32, 500, 151936) > w
    assert bp.policy_select_workspace_size(32, 2560, 2048, 9) >= 256 + 32 * 2048 * 4 + 64 * 2560 * 2
    assert lib.bp_spec_accept_workspace_size(-1, 0, 10) == 0


def _align(x, a=256):
    return (x + a - 1) // a * a


@pytest.mark.parametrize("s,td,vocab", [(1, 15, 151936), (1, 16, 151936), (4, 60, 32000), (5, 75, 32000),
                                        (2, 23, 151936), (3, 23, 151936), (1, 0, 5), (32, 470, 151936),
                                        (200000, 200000, 16), (9, 100, 16385)])
def test_acceptance_workspace_follows_the_path_choice(lib, s, td, vocab):
    """The workspace carries the throughput kernels' regions (chunk statistics, the totals of the
    draw's chunk parts (up to 4 per chunk), segment masses) exactly when either temperature takes
    those kernels: this pins the tests' mirror of the library's choice (accept_uses_batch) to the
    library, on the CPU."""
    from _gpu import accept_uses_batch

    blocks = (td + 1,) + (1,) * (s - 1)
    cluster = 256 + _align(4 * s) + _align(4 * td) + _align(4 * (td + s))
    chunks = -(-vocab // 16384)
    rows = 2 * td + s
    batch = _align(rows * chunks * 8) + _align(s * chunks * 4 * 16) + _align(s * chunks * 256 * 8)
    may = accept_uses_batch(blocks, vocab, 0.0) or accept_uses_batch(blocks, vocab, 1.0)
    assert bp.spec_accept_workspace_size(s, td, vocab) == cluster + (batch if may else 0)


def test_host_validation_needs_no_gpu(lib):
    vp = ctypes.c_void_p
    fake = vp(0x10000)
    ws = vp(0x20000)
    # NULL q
    rc = lib.bp_block_attention(None, fake, fake, fake, None, fake, fake, 1, 16, 2064, 16, 2064, 32, 8, 128, 1, 0,
                                0.0, ws, 4096, None)
    assert rc == 1
    # head ratio
    rc = lib.bp_block_attention(fake, fake, fake, fake, None, fake, fake, 1, 16, 2064, 16, 2064, 30, 8, 128, 1, 0,
                                0.0, ws, 4096, None)
    assert rc == 1
    # bf16 head_dim 64 is not implemented
    rc = lib.bp_block_attention(fake, fake, fake, fake, None, fake, fake, 1, 16, 2064, 16, 2064, 32, 8, 64, 1, 0,
                                0.0, ws, 4096, None)
    assert rc == 2
    # workspace too small / misaligned
    rc = lib.bp_block_attention(fake, fake, fake, fake, None, fake, fake, 1, 16, 2064, 16, 2064, 32, 8, 128, 1, 0,
                                0.0, ws, 16, None)
    assert rc == 4
    rc = lib.bp_block_attention(fake, fake, fake, fake, None, fake, fake, 1, 16, 2064, 16, 2064, 32, 8, 128, 1, 0,
                                0.0, vp(0x20010), 4096, None)
    assert rc == 4
    # acceptance: T > 0 without draft logits; negative temperature
    rc = lib.bp_spec_accept(fake, None, fake, fake, 1, 15, 1000, ctypes.c_float(1.0), fake, fake, fake, fake, None,
                            ws, 1 << 20, None)
    assert rc == 1
    rc = lib.bp_spec_accept(fake, fake, fake, fake, 1, 15, 1000, ctypes.c_float(-1.0), fake, fake, fake, fake, None,
                            ws, 1 << 20, None)
    assert rc == 1
    # policy: too many candidates
    rc = lib.bp_policy_select(fake, 64, None, 1, 64, fake, fake, 32, fake, fake, 65, fake, 1, None, fake, ws,
                              1 << 20, None)
    assert rc == 2



def test_paged_host_validation_needs_no_gpu(lib):
    vp, f32 = ctypes.c_void_p, ctypes.c_float
    fake, ws = vp(0x10000), vp(0x20000)

    def paged(block_table=fake, pps=33, page=64, pages=40, dtype=1, max_kv=2064):
        return lib.bp_block_attention_paged(fake, fake, fake, fake, None, fake, fake, block_table, pps, page, pages, 1,
                                            16, 2064, 16, max_kv, 32, 8, 128, dtype, 0, f32(0.0), ws, 4096, None)
    assert paged(block_table=None) == 1                       # no block table
    assert paged(page=24) == 1 and paged(page=8) == 1         # not a power of two >= 16
    assert paged(pps=32) == 1                                  # 32 pages of 64 < 2064 keys
    assert paged(dtype=0) == 2                                 # fp32 has no paged path

    def append(page=64, head_dim=128, dtype=1):
        return lib.bp_kv_append(fake, fake, fake, fake, fake, fake, fake, 33, page, 40, 1, 16, 8, head_dim, dtype, None)
    assert append(page=100) == 1
    assert append(head_dim=4) == 2                            # 8-byte rows: not a multiple of 16 bytes
    assert lib.bp_kv_append(fake, fake, fake, fake, fake, fake, None, 33, 64, 40, 1, 16, 8, 128, 1, None) == 1


def test_verify_epilogue_host_validation_needs_no_gpu(lib):
    vp, f32 = ctypes.c_void_p, ctypes.c_float
    fake, ws = vp(0x10000), vp(0x20000)

    def call(hidden=2560, vocab=151936, seqs=1, drafts=15, temp=1.0, h_draft=fake, ws_bytes=1 << 20, w=fake):
        return lib.bp_verify_epilogue(w, fake, h_draft, hidden, vocab, fake, fake, seqs, drafts, f32(temp), fake, fake,
                                      fake, fake, None, None, ws, ws_bytes, None)
    need = lib.bp_verify_epilogue_workspace_size(1, 15, 151936)
    assert 256 < need < (1 << 20) and need % 256 == 0
    assert call(w=None) == 1                      # no LM head
    assert call(temp=-1.0) == 1                   # negative temperature
    assert call(h_draft=None) == 1                # T > 0 needs the drafter's states
    assert call(hidden=100) == 2                  # hidden not a multiple of 64
    assert call(drafts=40, ws_bytes=need) == 4    # 81 rows: streamed, its workspace holds the logits
    big = lib.bp_verify_epilogue_workspace_size(1, 40, 151936)
    assert big >= 81 * 151936 * 4 + need and big % 256 == 0
    assert lib.bp_verify_epilogue_workspace_size(1, 15, 0) == 0   # no vocabulary
    assert call(w=vp(0x10008)) == 2               # LM head not 16-byte aligned
    assert call(ws_bytes=need - 256) == 4         # workspace too small
    assert call(seqs=0) == 0                      # nothing to do
    if not __import__("torch").cuda.is_available():
        assert call(temp=0.0, h_draft=None) == 3  # valid; no device to run on


def test_tau_select_host_validation_needs_no_gpu(lib):
    vp, f32 = ctypes.c_void_p, ctypes.c_float
    fake, ws = vp(0x10000), vp(0x20000)

    cands = (ctypes.c_int32 * 9)(*range(8, 25, 2))  # a host array

    def call(n=1000, jmax=24, nc=9, alpha=0.001, pred=fake, regret=fake, best=fake, cand=cands):
        return lib.bp_tau_select(fake, n, jmax, cand, nc, 16, f32(alpha), pred, fake, best, regret, fake, ws, 1 << 20,
                                 None)
    assert lib.bp_tau_select_workspace_size(1000) >= 256 + 4 * 8 * 4
    assert call(alpha=-1.0) == 1 and call(jmax=0) == 1 and call(best=None) == 1
    assert call(pred=None) == 1                  # a regret needs predicted sizes
    assert call(nc=33) == 2 and call(jmax=65) == 2
    assert call(n=0) == 0
    if not __import__("torch").cuda.is_available():
        assert call() == 3                         # valid; no device to run on
        assert call(jmax=20) == 1                  # candidate 22 beyond 20-position rows
        assert call(cand=(ctypes.c_int32 * 9)(8, 10, 12, 14, 16, 18, 20, 24, 22)) == 1  # not increasing


def test_verify_commit_host_validation_needs_no_gpu(lib):
    vp = ctypes.c_void_p
    fake, ws = vp(0x10000), vp(0x20000)

    def call(n=4, cap=4096, ctx=fake, cu_kv=fake, ws_bytes=256):
        return lib.bp_verify_commit(ctx, fake, fake, fake, n, cap, None, cu_kv, ws, ws_bytes, None)
    assert call(n=-1) == 1 and call(cap=0) == 1 and call(ctx=None) == 1 and call(cu_kv=None) == 1
    assert call(ws_bytes=128) == 4
    assert call(n=0) == 0
    if not __import__("torch").cuda.is_available():
        assert call() == 3


def test_no_cpu_fallback_without_gpu(lib):
    import torch

    if torch.cuda.is_available():
        pytest.skip("a GPU is present; this checks the GPU-less failure mode")
    vp = ctypes.c_void_p
    fake = vp(0x10000)
    rc = lib.bp_block_attention(fake, fake, fake, fake, None, fake, fake, 1, 16, 2064, 16, 2064, 32, 8, 128, 1, 0,
                                0.0, vp(0x20000), 4096, None)
    assert rc == 3  # BP_ERR_CUDA: there is nothing to fall back to


def test_product_package_never_imports_the_oracle():
    pkg = os.path.join(ROOT, "paper_2606_31315_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            path = os.path.join(dirpath, f)
            if f.endswith(".py"):
                tree = ast.parse(open(path).read())
                for node in ast.walk(tree):
                    if isinstance(node, ast.Import):
                        assert all(not a.name.startswith("oracle") for a in node.names), path
                    if isinstance(node, ast.ImportFrom):
                        assert not (node.module or "").startswith("oracle"), path
            if f.endswith((".cu", ".cuh", ".h")):
                assert "bpo_" not in open(path).read(), path


def test_build_compiles_every_source():
    """build() (the only build step on a fresh machine) compiles every CUDA source and tracks every
    header of csrc/: a file left off the lists would silently be missing from the library."""
    csrc = os.path.join(ROOT, "paper_2606_31315_gb300", "csrc")
    on_disk = sorted(f for f in os.listdir(csrc) if f.endswith(".cu"))
    headers = sorted(f for f in os.listdir(csrc) if f.endswith(".cuh"))
    assert sorted(_build.SOURCES) == on_disk
    assert sorted(_build.HEADERS) == headers


def test_noalloc_host_validation_needs_no_gpu(lib):
    """bp_spec_accept_noalloc checks its arguments as bp_spec_accept does, before touching CUDA."""
    vp, i32, f32 = ctypes.c_void_p, ctypes.c_int, ctypes.c_float
    lib.bp_spec_accept_noalloc.argtypes = [vp, vp, vp, vp, i32, i32, i32, f32, vp, vp, vp, vp, vp, vp, vp]
    lib.bp_spec_accept_noalloc.restype = i32
    fake = vp(0x10000)

    def call(target=fake, draft=fake, tokens=fake, cu=fake, s=1, td=15, vocab=1000, temp=1.0, ua=fake, us=fake,
             n_acc=fake, out=fake):
        return lib.bp_spec_accept_noalloc(target, draft, tokens, cu, s, td, vocab, f32(temp), ua, us, n_acc, out,
                                          None, None, None)
    assert call(s=0) == 0                            # nothing to compute
    assert call(s=-1) == 1 and call(td=-1) == 1 and call(vocab=0) == 1
    assert call(target=None) == 1 and call(cu=None) == 1 and call(n_acc=None) == 1 and call(out=None) == 1
    assert call(tokens=None) == 1                    # drafts without their tokens
    assert call(temp=-1.0) == 1 and call(temp=float("inf")) == 1
    assert call(us=None) == 1 and call(draft=None) == 1 and call(ua=None) == 1  # T > 0 needs them
    assert call(temp=0.0, draft=None, ua=None, us=None) == 3  # greedy needs none of them; then no device
    assert call(s=1 << 20, td=1 << 20, vocab=1 << 20) == 2   # more than 2^40 logits
    assert call() == 3                               # valid arguments, no sm_103 device: BP_ERR_CUDA
