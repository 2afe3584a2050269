"""ctypes binding of libblockpilot (argument marshalling only).

Every function takes CUDA tensors, passes their device pointers and the current torch
stream to the C ABI and returns the output tensors.  No step of the computation happens
here; if the library is missing or the call fails the binding raises -- there is no
fallback path.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np
import torch

from . import _build

BP_OK = 0
BP_ERR_INVALID_ARG = 1
BP_ERR_UNSUPPORTED = 2
BP_ERR_CUDA = 3
BP_ERR_WORKSPACE = 4
BP_ERR_TIMEOUT = 5
BP_ERR_DEVICE_FLAG = 6

MASK_CAUSAL = 0
MASK_BIDIR = 1
F32 = 0
BF16 = 1

_lib = None


class BlockPilotError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        msg = _lib.bp_error_string(status).decode() if _lib is not None else str(status)
        super().__init__(f"{where}: {msg}")


def library_path() -> str:
    return _build.LIB


def load():
    """Load libblockpilot.so (built by ``__graft_entry__.build()`` / ``_build.build()``)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(_build.LIB):
        raise RuntimeError(f"libblockpilot.so is not built ({_build.LIB}); run __graft_entry__.build() first")
    lib = ctypes.CDLL(_build.LIB)
    vp, i32, i64, f32, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_float, ctypes.c_size_t
    lib.bp_abi_version.argtypes = []
    lib.bp_abi_version.restype = i32
    lib.bp_error_string.argtypes = [i32]
    lib.bp_error_string.restype = ctypes.c_char_p
    lib.bp_block_attention_workspace_size.argtypes = [i32, i32, i32, i32, i32]
    lib.bp_block_attention_workspace_size.restype = sz
    lib.bp_block_attention.argtypes = [vp, vp, vp, vp, vp, vp, vp, i32, i32, i32, i32, i32, i32, i32, i32, i32, i32,
                                       f32, vp, sz, vp]
    lib.bp_block_attention.restype = i32
    lib.bp_block_attention_paged.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp, i32, i32, i32, i32, i32, i32, i32, i32,
                                             i32, i32, i32, i32, i32, f32, vp, sz, vp]
    lib.bp_block_attention_paged.restype = i32
    lib.bp_kv_append.argtypes = [vp, vp, vp, vp, vp, vp, vp, i32, i32, i32, i32, i32, i32, i32, i32, vp]
    lib.bp_kv_append.restype = i32
    lib.bp_spec_accept_workspace_size.argtypes = [i32, i32, i32]
    lib.bp_spec_accept_workspace_size.restype = sz
    lib.bp_spec_accept.argtypes = [vp, vp, vp, vp, i32, i32, i32, f32, vp, vp, vp, vp, vp, vp, sz, vp]
    lib.bp_spec_accept.restype = i32
    lib.bp_policy_select_workspace_size.argtypes = [i32, i32, i32, i32]
    lib.bp_policy_select_workspace_size.restype = sz
    lib.bp_policy_select.argtypes = [vp, i64, vp, i32, i32, vp, vp, i32, vp, vp, i32, vp, i32, vp, vp, vp, sz, vp]
    lib.bp_policy_select.restype = i32
    lib.bp_verify_epilogue_workspace_size.argtypes = [i32, i32, i32]
    lib.bp_verify_epilogue_workspace_size.restype = sz
    lib.bp_verify_epilogue.argtypes = [vp, vp, vp, i32, i32, vp, vp, i32, i32, f32, vp, vp, vp, vp, vp, vp, vp, sz,
                                       vp]
    lib.bp_verify_epilogue.restype = i32
    lib.bp_tau_select_workspace_size.argtypes = [i32]
    lib.bp_tau_select_workspace_size.restype = sz
    lib.bp_tau_select.argtypes = [vp, i32, i32, vp, i32, i32, f32, vp, vp, vp, vp, vp, vp, sz, vp]
    lib.bp_tau_select.restype = i32
    lib.bp_verify_commit.argtypes = [vp, vp, vp, vp, i32, i32, vp, vp, vp, sz, vp]
    lib.bp_verify_commit.restype = i32
    lib.bp_get_status.argtypes = [vp, vp]
    lib.bp_get_status.restype = i32
    _lib = lib
    return lib


def _ptr(t) -> ctypes.c_void_p | None:
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _check(rc: int, where: str):
    if rc != BP_OK:
        raise BlockPilotError(rc, where)


def _cuda(t, name):
    if t is not None and (not t.is_cuda or not t.is_contiguous()):
        raise ValueError(f"{name} must be a contiguous CUDA tensor")


def workspace(nbytes: int, device) -> torch.Tensor:
    """Zero-filled device workspace (the library itself never allocates)."""
    return torch.zeros(max(int(nbytes), 256), dtype=torch.uint8, device=device)


# --------------------------------------------------------------------------- attention
def block_attention_workspace_size(num_seqs, max_q_len, num_q_heads, num_kv_heads, head_dim) -> int:
    return int(load().bp_block_attention_workspace_size(num_seqs, max_q_len, num_q_heads, num_kv_heads, head_dim))


def block_attention(q, k, v, cu_q, cu_kv, max_q_len: int, max_kv_len: int, mask: int = MASK_CAUSAL,
                    softmax_scale: float = 0.0, out=None, lse=None, ws=None, stream=None):
    """O = block attention of q over (k, v); see ``bp_block_attention`` in include/blockpilot.h.

    q [total_q, Hq, D], k/v [total_kv, Hkv, D] (bf16 or fp32), cu_q/cu_kv int32 [S+1] on the device.
    Returns (o, lse_or_None)."""
    lib = load()
    for t, n in ((q, "q"), (k, "k"), (v, "v"), (cu_q, "cu_q"), (cu_kv, "cu_kv"), (out, "out"), (lse, "lse")):
        _cuda(t, n)
    dtype = {torch.bfloat16: BF16, torch.float32: F32}.get(q.dtype)
    if dtype is None or k.dtype != q.dtype or v.dtype != q.dtype:
        raise ValueError("q, k, v must all be bf16 or all fp32")
    total_q, hq, d = q.shape
    total_kv, hkv, _ = k.shape
    s = cu_q.numel() - 1
    if out is None:
        out = torch.empty_like(q)
    if ws is None:
        ws = workspace(lib.bp_block_attention_workspace_size(s, max_q_len, hq, hkv, d), q.device)
    rc = lib.bp_block_attention(_ptr(q), _ptr(k), _ptr(v), _ptr(out), _ptr(lse), _ptr(cu_q), _ptr(cu_kv), s, total_q,
                                total_kv, int(max_q_len), int(max_kv_len), hq, hkv, d, dtype, int(mask),
                                float(softmax_scale), _ptr(ws), ws.numel(), _stream(stream))
    _check(rc, "bp_block_attention")
    return out, lse


def block_attention_paged(q, k_cache, v_cache, cu_q, cu_kv, block_table, page_size: int, total_kv: int,
                          max_q_len: int, max_kv_len: int, mask: int = MASK_CAUSAL, softmax_scale: float = 0.0,
                          out=None, lse=None, ws=None, stream=None):
    """Block attention over a paged KV cache; see ``bp_block_attention_paged`` in include/blockpilot.h.

    q [total_q, Hq, 128] bf16; k_cache/v_cache [num_pages * page_size, Hkv, 128] bf16; block_table int32
    [S, pages_per_seq]; cu_q/cu_kv int32 [S+1] on the device; total_kv = cu_kv[S].  Returns (o, lse_or_None)."""
    lib = load()
    for t, n in ((q, "q"), (k_cache, "k_cache"), (v_cache, "v_cache"), (cu_q, "cu_q"), (cu_kv, "cu_kv"),
                 (block_table, "block_table"), (out, "out"), (lse, "lse")):
        _cuda(t, n)
    dtype = {torch.bfloat16: BF16, torch.float32: F32}.get(q.dtype)
    if dtype is None or k_cache.dtype != q.dtype or v_cache.dtype != q.dtype:
        raise ValueError("q, k_cache, v_cache must share one dtype")
    total_q, hq, d = q.shape
    pool_rows, hkv, _ = k_cache.shape
    s = cu_q.numel() - 1
    if out is None:
        out = torch.empty_like(q)
    if ws is None:
        ws = workspace(lib.bp_block_attention_workspace_size(s, max_q_len, hq, hkv, d), q.device)
    rc = lib.bp_block_attention_paged(_ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(out), _ptr(lse), _ptr(cu_q),
                                      _ptr(cu_kv), _ptr(block_table), block_table.shape[1], int(page_size),
                                      pool_rows // int(page_size), s, total_q, int(total_kv), int(max_q_len),
                                      int(max_kv_len), hq, hkv, d, dtype, int(mask), float(softmax_scale), _ptr(ws),
                                      ws.numel(), _stream(stream))
    _check(rc, "bp_block_attention_paged")
    return out, lse


def kv_append(k_cache, v_cache, k_new, v_new, cu_new, cu_kv, block_table, page_size: int, stream=None):
    """Writes each sequence's new K/V rows into its pages; see ``bp_kv_append``."""
    lib = load()
    for t, n in ((k_cache, "k_cache"), (v_cache, "v_cache"), (k_new, "k_new"), (v_new, "v_new"), (cu_new, "cu_new"),
                 (cu_kv, "cu_kv"), (block_table, "block_table")):
        _cuda(t, n)
    dtype = {torch.bfloat16: BF16, torch.float32: F32}.get(k_new.dtype)
    if dtype is None or any(t.dtype != k_new.dtype for t in (k_cache, v_cache, v_new)):
        raise ValueError("caches and new rows must share one dtype (bf16 or fp32)")
    total_new, hkv, d = k_new.shape
    rc = lib.bp_kv_append(_ptr(k_cache), _ptr(v_cache), _ptr(k_new), _ptr(v_new), _ptr(cu_new), _ptr(cu_kv),
                          _ptr(block_table), block_table.shape[1], int(page_size), k_cache.shape[0] // int(page_size),
                          cu_new.numel() - 1, total_new, hkv, d, dtype, _stream(stream))
    _check(rc, "bp_kv_append")


# --------------------------------------------------------------------------- acceptance
def spec_accept_workspace_size(num_seqs, total_draft, vocab) -> int:
    return int(load().bp_spec_accept_workspace_size(num_seqs, total_draft, vocab))


def spec_accept(target_logits, draft_logits, draft_tokens, cu_draft, temperature: float, u_accept=None,
                u_sample=None, n_accepted=None, out_tokens=None, accept_prob=None, want_accept_prob=True, ws=None,
                stream=None):
    """Lossless acceptance; see ``bp_spec_accept``.  Returns (n_accepted, out_tokens, accept_prob)."""
    lib = load()
    for t, n in ((target_logits, "target_logits"), (draft_logits, "draft_logits"), (draft_tokens, "draft_tokens"),
                 (cu_draft, "cu_draft"), (u_accept, "u_accept"), (u_sample, "u_sample")):
        _cuda(t, n)
    s = cu_draft.numel() - 1
    total_draft = draft_tokens.numel()
    vocab = target_logits.shape[1]
    dev = target_logits.device
    if n_accepted is None:
        n_accepted = torch.empty(s, dtype=torch.int32, device=dev)
    if out_tokens is None:
        out_tokens = torch.empty(total_draft + s, dtype=torch.int32, device=dev)
    if accept_prob is None and want_accept_prob:
        accept_prob = torch.empty(total_draft, dtype=torch.float32, device=dev)
    if ws is None:
        ws = workspace(lib.bp_spec_accept_workspace_size(s, total_draft, vocab), dev)
    rc = lib.bp_spec_accept(_ptr(target_logits), _ptr(draft_logits), _ptr(draft_tokens), _ptr(cu_draft), s,
                            total_draft, vocab, float(temperature), _ptr(u_accept), _ptr(u_sample), _ptr(n_accepted),
                            _ptr(out_tokens), _ptr(accept_prob), _ptr(ws), ws.numel(), _stream(stream))
    _check(rc, "bp_spec_accept")
    return n_accepted, out_tokens, accept_prob


# --------------------------------------------------------------------------- verify epilogue
def verify_epilogue_workspace_size(num_seqs, total_draft, vocab) -> int:
    return int(load().bp_verify_epilogue_workspace_size(num_seqs, total_draft, vocab))


def verify_epilogue(lm_head, h_target, h_draft, draft_tokens, cu_draft, temperature: float, u_accept=None,
                    u_sample=None, n_accepted=None, out_tokens=None, accept_prob=None, want_accept_prob=True,
                    logits_out=None, ws=None, stream=None):
    """LM head fused with the lossless acceptance; see ``bp_verify_epilogue``.  Returns
    (n_accepted, out_tokens, accept_prob)."""
    lib = load()
    for t, n in ((lm_head, "lm_head"), (h_target, "h_target"), (h_draft, "h_draft"), (draft_tokens, "draft_tokens"),
                 (cu_draft, "cu_draft"), (u_accept, "u_accept"), (u_sample, "u_sample"), (logits_out, "logits_out")):
        _cuda(t, n)
    if lm_head.dtype != torch.bfloat16 or h_target.dtype != torch.bfloat16:
        raise TypeError("verify_epilogue: lm_head and the hidden states must be bf16")
    s = cu_draft.numel() - 1
    total_draft = draft_tokens.numel()
    vocab, hidden = lm_head.shape
    dev = lm_head.device
    if n_accepted is None:
        n_accepted = torch.empty(s, dtype=torch.int32, device=dev)
    if out_tokens is None:
        out_tokens = torch.empty(total_draft + s, dtype=torch.int32, device=dev)
    if accept_prob is None and want_accept_prob:
        accept_prob = torch.empty(total_draft, dtype=torch.float32, device=dev)
    if ws is None:
        ws = workspace(lib.bp_verify_epilogue_workspace_size(s, total_draft, vocab), dev)
    rc = lib.bp_verify_epilogue(_ptr(lm_head), _ptr(h_target), _ptr(h_draft), hidden, vocab, _ptr(draft_tokens),
                                _ptr(cu_draft), s, total_draft, float(temperature), _ptr(u_accept), _ptr(u_sample),
                                _ptr(n_accepted), _ptr(out_tokens), _ptr(accept_prob), _ptr(logits_out), _ptr(ws),
                                ws.numel(), _stream(stream))
    _check(rc, "bp_verify_epilogue")
    return n_accepted, out_tokens, accept_prob


# --------------------------------------------------------------------------- decoding-loop commit
def verify_commit(ctx_lens, n_accepted, out_tokens, cu_draft, capacity: int, anchor=None, cu_kv_next=None, ws=None,
                  stream=None):
    """Device-side commit of a verify step; see ``bp_verify_commit``.  ctx_lens is updated in place.
    Returns (anchor, cu_kv_next)."""
    lib = load()
    for t, n in ((ctx_lens, "ctx_lens"), (n_accepted, "n_accepted"), (out_tokens, "out_tokens"),
                 (cu_draft, "cu_draft"), (anchor, "anchor"), (cu_kv_next, "cu_kv_next")):
        _cuda(t, n)
    s = ctx_lens.numel()
    dev = ctx_lens.device
    if cu_kv_next is None:
        cu_kv_next = torch.empty(s + 1, dtype=torch.int32, device=dev)
    if ws is None:
        ws = workspace(256, dev)
    rc = lib.bp_verify_commit(_ptr(ctx_lens), _ptr(n_accepted), _ptr(out_tokens), _ptr(cu_draft), s, int(capacity),
                              _ptr(anchor), _ptr(cu_kv_next), _ptr(ws), ws.numel(), _stream(stream))
    _check(rc, "bp_verify_commit")
    return anchor, cu_kv_next


# --------------------------------------------------------------------------- acceptance-length model
def tau_select_workspace_size(num_reqs) -> int:
    return int(load().bp_tau_select_workspace_size(num_reqs))


def tau_select(gamma, candidates, train_block: int, alpha: float, predicted=None, tau=None, best=None, regret=None,
               summary=None, want_tau=True, ws=None, stream=None):
    """Appendix A's tau(b; x), B*(x) and regret; see ``bp_tau_select``.  candidates is a host
    sequence (list, numpy array or CPU tensor).  Returns (tau, best, regret, summary)."""
    lib = load()
    for t, n in ((gamma, "gamma"), (predicted, "predicted")):
        _cuda(t, n)
    g = gamma if gamma.dim() == 2 else gamma.reshape(-1, 1)
    n, jmax = g.shape
    cand = np.ascontiguousarray(candidates.cpu().numpy() if torch.is_tensor(candidates) else candidates,
                                dtype=np.int32)  # a host array
    nc = cand.size
    dev = gamma.device
    if tau is None and want_tau:
        tau = torch.empty(n, nc, dtype=torch.float32, device=dev)
    if best is None:
        best = torch.empty(n, dtype=torch.int32, device=dev)
    if regret is None and predicted is not None:
        regret = torch.empty(n, dtype=torch.float32, device=dev)
    if summary is None:
        summary = torch.empty(4, dtype=torch.float64, device=dev)
    if ws is None:
        ws = workspace(lib.bp_tau_select_workspace_size(n), dev)
    rc = lib.bp_tau_select(_ptr(g), n, jmax, cand.ctypes.data, nc, int(train_block), float(alpha), _ptr(predicted),
                           _ptr(tau), _ptr(best), _ptr(regret), _ptr(summary), _ptr(ws), ws.numel(), _stream(stream))
    _check(rc, "bp_tau_select")
    return tau, best, regret, summary


# --------------------------------------------------------------------------- policy head
def policy_select_workspace_size(num_reqs, d_in, hidden, num_cand) -> int:
    return int(load().bp_policy_select_workspace_size(num_reqs, d_in, hidden, num_cand))


def policy_select(feats, w1, b1, w2, b2, candidates, row_index=None, num_reqs=None, block_size=None, logits=None,
                  want_logits=True, ws=None, stream=None):
    """Block-size policy head; see ``bp_policy_select``.  Returns (block_size, logits)."""
    lib = load()
    for t, n in ((feats, "feats"), (w1, "w1"), (b1, "b1"), (w2, "w2"), (b2, "b2"), (candidates, "candidates"),
                 (row_index, "row_index")):
        _cuda(t, n)
    wdtype = {torch.bfloat16: BF16, torch.float32: F32}.get(w1.dtype)
    if wdtype is None or feats.dtype != w1.dtype or w2.dtype != w1.dtype:
        raise ValueError("feats, w1, w2 must share one dtype (bf16 or fp32)")
    hidden, d_in = w1.shape
    c = w2.shape[0]
    n = num_reqs if num_reqs is not None else (row_index.numel() if row_index is not None else feats.shape[0])
    dev = feats.device
    if block_size is None:
        block_size = torch.empty(n, dtype=torch.int32, device=dev)
    if logits is None and want_logits:
        logits = torch.empty((n, c), dtype=torch.float32, device=dev)
    if ws is None:
        ws = workspace(lib.bp_policy_select_workspace_size(n, d_in, hidden, c), dev)
    rc = lib.bp_policy_select(_ptr(feats), feats.stride(0), _ptr(row_index), n, d_in, _ptr(w1), _ptr(b1), hidden,
                              _ptr(w2), _ptr(b2), c, _ptr(candidates), wdtype, _ptr(logits), _ptr(block_size),
                              _ptr(ws), ws.numel(), _stream(stream))
    _check(rc, "bp_policy_select")
    return block_size, logits


def get_status(ws, stream=None) -> int:
    """Reads and clears the device error word of a workspace (synchronizes the stream)."""
    return int(load().bp_get_status(_ptr(ws), _stream(stream)))
