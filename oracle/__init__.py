"""BlockPilot fp64 CPU oracle -- test infrastructure only.

A plain, slow restatement of the block-verify hot path (block attention, lossless
speculative acceptance, block-size policy head, the LM-head projection that
feeds the acceptance, Appendix A's acceptance-length model, and the commit of the
decoding loop) written from the paper, in fp64.
Only the tests, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline leg
may import this package; the product path never does.  It shares no code with the
CUDA library.  The arithmetic lives in ``bpo.c``; this module only marshals numpy
arrays into it.

Every function here is pinned by ``tests/test_oracle_*.py`` to closed forms,
invariants and brute-force restatements (see each test's docstring).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import sys

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "bpo.c")
_LIB = os.path.join(_HERE, "libbpo_oracle.so")

MASK_CAUSAL = 0
MASK_BIDIR = 1

_lib = None


def build(force: bool = False) -> str:
    """Compile ``bpo.c`` into ``libbpo_oracle.so`` next to it (gcc, OpenMP)."""
    if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
        return _LIB
    tmp = _LIB + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB)
        dp = ctypes.POINTER(ctypes.c_double)
        ip = ctypes.POINTER(ctypes.c_int32)
        lib.bpo_block_attention.argtypes = [dp, dp, dp, dp, dp, ip, ip, ctypes.c_int, ctypes.c_int,
                                            ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_double]
        lib.bpo_block_attention.restype = ctypes.c_int
        lib.bpo_spec_accept.argtypes = [dp, dp, ip, ip, ctypes.c_int, ctypes.c_int, ctypes.c_double,
                                        dp, dp, ip, ip, dp, dp, dp]
        lib.bpo_spec_accept.restype = ctypes.c_int
        lib.bpo_policy_select.argtypes = [dp, ctypes.c_long, ip, ctypes.c_int, ctypes.c_int, dp, dp,
                                          ctypes.c_int, dp, dp, ctypes.c_int, ip, dp, ip, dp]
        lib.bpo_policy_select.restype = ctypes.c_int
        u16 = ctypes.POINTER(ctypes.c_uint16)
        lib.bpo_lm_head_logits.argtypes = [u16, u16, ctypes.c_int, ctypes.c_int, ctypes.c_int, dp, dp]
        lib.bpo_lm_head_logits.restype = ctypes.c_int
        lib.bpo_tau_select.argtypes = [dp, ctypes.c_int, ctypes.c_int, ip, ctypes.c_int, ctypes.c_int,
                                       ctypes.c_double, ip, dp, ip, dp, dp, dp]
        lib.bpo_tau_select.restype = ctypes.c_int
        lib.bpo_verify_commit.argtypes = [ip, ip, ip, ip, ctypes.c_int, ctypes.c_int, ip, ip]
        lib.bpo_verify_commit.restype = ctypes.c_int
        lib.bpo_num_threads.argtypes = []
        lib.bpo_num_threads.restype = ctypes.c_int
        lib.bpo_set_num_threads.argtypes = [ctypes.c_int]
        lib.bpo_set_num_threads.restype = None
        _lib = lib
    return _lib


def _f64(a):
    return None if a is None else np.ascontiguousarray(a, dtype=np.float64)


def _i32(a):
    return None if a is None else np.ascontiguousarray(a, dtype=np.int32)


def _p(a, ctype):
    return None if a is None else a.ctypes.data_as(ctypes.POINTER(ctype))


def num_threads() -> int:
    """OpenMP threads the oracle's parallel loops use."""
    return int(_load().bpo_num_threads())


def set_num_threads(n: int) -> None:
    """Thread count of the oracle's parallel loops from now on (timing only; results do not change)."""
    _load().bpo_set_num_threads(int(n))


def block_attention(q, k, v, cu_q, cu_kv, num_kv_heads: int, mask: int, scale: float | None = None):
    """Block attention (causal or bidirectional within the block) over a ragged KV cache.

    q: [total_q, Hq, D]; k, v: [total_kv, Hkv, D]; cu_q, cu_kv: [S+1] offsets.
    Returns (o [total_q, Hq, D], lse [total_q, Hq]) in fp64.
    """
    q, k, v = _f64(q), _f64(k), _f64(v)
    cu_q, cu_kv = _i32(cu_q), _i32(cu_kv)
    total_q, hq, d = q.shape
    if scale is None:
        scale = 1.0 / np.sqrt(d)
    o = np.zeros_like(q)
    lse = np.zeros((total_q, hq), dtype=np.float64)
    rc = _load().bpo_block_attention(_p(q, ctypes.c_double), _p(k, ctypes.c_double), _p(v, ctypes.c_double),
                                     _p(o, ctypes.c_double), _p(lse, ctypes.c_double),
                                     _p(cu_q, ctypes.c_int32), _p(cu_kv, ctypes.c_int32),
                                     len(cu_q) - 1, hq, int(num_kv_heads), d, int(mask), float(scale))
    if rc != 0:
        raise ValueError(f"oracle block_attention rejected its arguments (rc={rc})")
    return o, lse


def spec_accept(target_logits, draft_logits, draft_tokens, cu_draft, temperature: float,
                u_accept=None, u_sample=None):
    """Lossless speculative acceptance over the full vocabulary.

    target_logits: [total_draft + S, V]; draft_logits: [total_draft, V] (None at T=0);
    draft_tokens: [total_draft]; cu_draft: [S+1].
    Returns dict(n_accepted [S], out_tokens [total_draft+S], accept_prob [total_draft],
    ratio_margin [S], cdf_margin [S]).
    """
    t = _f64(target_logits)
    dl = _f64(draft_logits)
    x = _i32(draft_tokens)
    cu = _i32(cu_draft)
    ua, us = _f64(u_accept), _f64(u_sample)
    s = len(cu) - 1
    vocab = t.shape[1]
    total_draft = int(cu[-1])
    n_acc = np.zeros(s, dtype=np.int32)
    out = np.zeros(total_draft + s, dtype=np.int32)
    ap = np.zeros(total_draft, dtype=np.float64)
    rm = np.zeros(s, dtype=np.float64)
    cm = np.zeros(s, dtype=np.float64)
    dp = ctypes.c_double
    rc = _load().bpo_spec_accept(_p(t, dp), _p(dl, dp), _p(x, ctypes.c_int32), _p(cu, ctypes.c_int32), s, vocab,
                                 float(temperature), _p(ua, dp), _p(us, dp), _p(n_acc, ctypes.c_int32),
                                 _p(out, ctypes.c_int32), _p(ap, dp), _p(rm, dp), _p(cm, dp))
    if rc != 0:
        raise ValueError(f"oracle spec_accept rejected its arguments (rc={rc})")
    return dict(n_accepted=n_acc, out_tokens=out, accept_prob=ap, ratio_margin=rm, cdf_margin=cm)


def policy_select(feats, w1, b1, w2, b2, candidates, row_index=None):
    """Block-size policy head: B_hat = candidates[argmax(W2 relu(W1 x + b1) + b2)].

    feats: [rows, d_in]; w1: [H, d_in]; b1: [H]; w2: [C, H]; b2: [C]; candidates: [C].
    Returns dict(block_size [N], logits [N, C], top2_margin [N]).
    """
    f = _f64(feats)
    w1, b1, w2, b2 = _f64(w1), _f64(b1), _f64(w2), _f64(b2)
    cand = _i32(candidates)
    ri = _i32(row_index)
    n = len(ri) if ri is not None else f.shape[0]
    hidden, d_in = w1.shape
    c = w2.shape[0]
    bs = np.zeros(n, dtype=np.int32)
    lo = np.zeros((n, c), dtype=np.float64)
    mg = np.zeros(n, dtype=np.float64)
    dp = ctypes.c_double
    rc = _load().bpo_policy_select(_p(f, dp), f.shape[1], _p(ri, ctypes.c_int32), n, d_in, _p(w1, dp),
                                   _p(b1, dp), hidden, _p(w2, dp), _p(b2, dp), c, _p(cand, ctypes.c_int32),
                                   _p(lo, dp), _p(bs, ctypes.c_int32), _p(mg, dp))
    if rc != 0:
        raise ValueError(f"oracle policy_select rejected its arguments (rc={rc})")
    return dict(block_size=bs, logits=lo, top2_margin=mg)



def lm_head_logits(w_bits, h_bits, with_abs: bool = False):
    """fp64 logits = h @ W^T of bf16 operands given as uint16 bits.

    w_bits: [V, H]; h_bits: [rows, H].  Returns logits [rows, V] (and, with with_abs,
    sum_k |W[v,k] h[r,k]| of the same shape, the scale of any fp32 rounding error).
    """
    w = np.ascontiguousarray(w_bits, dtype=np.uint16)
    h = np.ascontiguousarray(h_bits, dtype=np.uint16).reshape(-1, w.shape[1])
    rows, (vocab, hidden) = h.shape[0], w.shape
    out = np.zeros((rows, vocab), dtype=np.float64)
    mag = np.zeros((rows, vocab), dtype=np.float64) if with_abs else None
    u16 = ctypes.c_uint16
    rc = _load().bpo_lm_head_logits(_p(w, u16), _p(h, u16), rows, vocab, hidden, _p(out, ctypes.c_double),
                                    _p(mag, ctypes.c_double))
    if rc != 0:
        raise ValueError(f"oracle lm_head_logits rejected its arguments (rc={rc})")
    return (out, mag) if with_abs else out


def verify_epilogue(w_bits, h_target_bits, h_draft_bits, draft_tokens, cu_draft, temperature: float,
                    u_accept=None, u_sample=None, with_abs: bool = False):
    """The verify step from final hidden states: LM-head logits of the target rows (and, at
    T > 0, of the drafter's rows) followed by the lossless acceptance over them.

    Returns spec_accept's dict plus target_logits / draft_logits (fp64) and, with with_abs,
    target_abs / draft_abs (the error scales of lm_head_logits).
    """
    greedy = temperature == 0.0
    t = lm_head_logits(w_bits, h_target_bits, with_abs)
    d = None if greedy or h_draft_bits is None else lm_head_logits(w_bits, h_draft_bits, with_abs)
    tl, ta = t if with_abs else (t, None)
    dl, da = (d if with_abs else (d, None)) if d is not None else (None, None)
    res = spec_accept(tl, dl, draft_tokens, cu_draft, temperature, u_accept, u_sample)
    res.update(target_logits=tl, draft_logits=dl)
    if with_abs:
        res.update(target_abs=ta, draft_abs=da)
    return res



def tau_select(gamma, candidates, train_block: int, alpha: float, predicted=None):
    """Appendix A: tau(b; x) for every candidate b, B*(x), and (given predicted B_hat) the regret.

    gamma: [n, jmax] per-position predictability (jmax == 1: one gamma_x per request, geometric
    form).  Returns dict(tau [n, C], best [n], regret [n] or None, lips [n], summary [4] =
    (mean regret, mean |B* - B_hat|, L_tau, L_tau * mean |B* - B_hat|)).
    """
    g = np.ascontiguousarray(gamma, dtype=np.float64)
    if g.ndim == 1:
        g = g[:, None]
    cand = _i32(candidates)
    pred = _i32(predicted)
    n, jmax = g.shape
    tau = np.zeros((n, len(cand)), dtype=np.float64)
    best = np.zeros(n, dtype=np.int32)
    regret = np.zeros(n, dtype=np.float64) if pred is not None else None
    lips = np.zeros(n, dtype=np.float64)
    summary = np.zeros(4, dtype=np.float64)
    dp, ip = ctypes.c_double, ctypes.c_int32
    rc = _load().bpo_tau_select(_p(g, dp), n, jmax, _p(cand, ip), len(cand), int(train_block), float(alpha),
                                _p(pred, ip), _p(tau, dp), _p(best, ip), _p(regret, dp), _p(lips, dp),
                                _p(summary, dp))
    if rc != 0:
        raise ValueError(f"oracle tau_select rejected its arguments (rc={rc})")
    return dict(tau=tau, best=best, regret=regret, lips=lips, summary=summary)



def verify_commit(ctx, n_accepted, out_tokens, cu_draft, capacity: int):
    """The decoding loop's commit after a verify step: new context lengths (anchor + accepted drafts
    stay), the next anchors and the next pass's key offsets.  Returns dict(ctx, anchor, cu_kv)."""
    c = np.array(ctx, dtype=np.int32)
    n = _i32(n_accepted)
    out = _i32(out_tokens)
    cu = _i32(cu_draft)
    s = len(c)
    anchor = np.zeros(s, dtype=np.int32)
    cu_kv = np.zeros(s + 1, dtype=np.int32)
    ip = ctypes.c_int32
    rc = _load().bpo_verify_commit(_p(c, ip), _p(n, ip), _p(out, ip), _p(cu, ip), s, int(capacity), _p(anchor, ip),
                                   _p(cu_kv, ip))
    if rc != 0:
        raise ValueError(f"oracle verify_commit rejected its arguments (rc={rc})")
    return dict(ctx=c, anchor=anchor, cu_kv=cu_kv)


if __name__ == "__main__":  # pragma: no cover
    print(build(force="--force" in sys.argv))
