"""Pins for the oracle's block attention (CPU only).

The oracle is checked against things other than itself:
  * brute force: the full masked score matrix with -inf entries, softmax by numpy;
  * the textbook single-token decode (B = 1 is plain decode attention);
  * invariants: causal and bidirectional rows agree on the last block row, a causal
    row i equals a decode over the first L + i + 1 keys, GQA equals MHA with repeated
    KV heads, bidirectional output is invariant under a permutation of the keys,
    constant V rows give that constant back (outputs are convex combinations).
A dropped mask term, an off-by-one in the causal limit, a wrong KV-head mapping, a
missing scale or a transposed operand each fail at least one of these.
"""
import numpy as np
import pytest

from paper_2606_31315_gb300 import workloads as wl

CAUSAL, BIDIR = 0, 1


def _problem(seed, ctx, block, hq=4, hkv=2, d=16):
    rng = np.random.default_rng(seed)
    cu_q = wl.offsets(block)
    cu_kv = wl.offsets(np.asarray(ctx) + np.asarray(block))
    q = rng.standard_normal((cu_q[-1], hq, d))
    k = rng.standard_normal((cu_kv[-1], hkv, d))
    v = rng.standard_normal((cu_kv[-1], hkv, d))
    return q, k, v, cu_q, cu_kv


def _brute(q, k, v, cu_q, cu_kv, hkv, mask, scale):
    hq, d = q.shape[1], q.shape[2]
    g = hq // hkv
    o = np.zeros_like(q)
    lse = np.zeros(q.shape[:2])
    for s in range(len(cu_q) - 1):
        B = cu_q[s + 1] - cu_q[s]
        nkv = cu_kv[s + 1] - cu_kv[s]
        L = nkv - B
        qs, ks, vs = q[cu_q[s]:cu_q[s + 1]], k[cu_kv[s]:cu_kv[s + 1]], v[cu_kv[s]:cu_kv[s + 1]]
        allowed = np.ones((B, nkv), dtype=bool)
        if mask == CAUSAL:
            allowed = np.arange(nkv)[None, :] <= (L + np.arange(B))[:, None]
        for h in range(hq):
            S = scale * (qs[:, h, :] @ ks[:, h // g, :].T)
            S = np.where(allowed, S, -np.inf)
            m = S.max(axis=1, keepdims=True)
            E = np.exp(S - m)
            Z = E.sum(axis=1, keepdims=True)
            o[cu_q[s]:cu_q[s + 1], h, :] = (E / Z) @ vs[:, h // g, :]
            lse[cu_q[s]:cu_q[s + 1], h] = (m + np.log(Z))[:, 0]
    return o, lse


@pytest.mark.parametrize("mask", [CAUSAL, BIDIR])
def test_matches_bruteforce_masked_matrix(oracle_mod, mask):
    q, k, v, cu_q, cu_kv = _problem(1, ctx=[5, 0, 13], block=[3, 4, 1], hq=6, hkv=2, d=8)
    scale = 0.37
    o, lse = oracle_mod.block_attention(q, k, v, cu_q, cu_kv, 2, mask, scale)
    ob, lseb = _brute(q, k, v, cu_q, cu_kv, 2, mask, scale)
    np.testing.assert_allclose(o, ob, rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse, lseb, rtol=0, atol=1e-12)


def test_block_of_one_is_plain_decode(oracle_mod):
    q, k, v, cu_q, cu_kv = _problem(2, ctx=[20], block=[1], hq=4, hkv=4, d=32)
    for mask in (CAUSAL, BIDIR):
        o, _ = oracle_mod.block_attention(q, k, v, cu_q, cu_kv, 4, mask)
        for h in range(4):
            # textbook decode: softmax(q K^T / sqrt(d)) V
            sc = k[:, h, :] @ q[0, h, :] / np.sqrt(32)
            w = np.exp(sc - sc.max())
            w /= w.sum()
            np.testing.assert_allclose(o[0, h], w @ v[:, h, :], rtol=0, atol=1e-12)


def test_causal_and_bidir_agree_on_last_row(oracle_mod):
    q, k, v, cu_q, cu_kv = _problem(3, ctx=[7, 11], block=[5, 2])
    oc, lc = oracle_mod.block_attention(q, k, v, cu_q, cu_kv, 2, CAUSAL)
    ob, lb = oracle_mod.block_attention(q, k, v, cu_q, cu_kv, 2, BIDIR)
    last = cu_q[1:] - 1
    np.testing.assert_array_equal(oc[last], ob[last])
    np.testing.assert_array_equal(lc[last], lb[last])
    # and differ elsewhere (the masks are not the same)
    assert np.abs(oc[0] - ob[0]).max() > 1e-3


def test_causal_row_is_decode_over_prefix(oracle_mod):
    L, B = 9, 6
    q, k, v, cu_q, cu_kv = _problem(4, ctx=[L], block=[B], hq=4, hkv=2, d=16)
    oc, _ = oracle_mod.block_attention(q, k, v, cu_q, cu_kv, 2, CAUSAL)
    for i in range(B):
        n = L + i + 1
        od, _ = oracle_mod.block_attention(q[i:i + 1], k[:n], v[:n], [0, 1], [0, n], 2, CAUSAL)
        np.testing.assert_allclose(oc[i], od[0], rtol=0, atol=1e-13)


def test_gqa_equals_mha_with_repeated_kv(oracle_mod):
    q, k, v, cu_q, cu_kv = _problem(5, ctx=[6, 3], block=[4, 5], hq=8, hkv=2, d=8)
    g = 4
    for mask in (CAUSAL, BIDIR):
        o1, l1 = oracle_mod.block_attention(q, k, v, cu_q, cu_kv, 2, mask)
        o2, l2 = oracle_mod.block_attention(q, np.repeat(k, g, axis=1), np.repeat(v, g, axis=1), cu_q, cu_kv, 8,
                                            mask)
        np.testing.assert_allclose(o1, o2, rtol=0, atol=1e-14)
        np.testing.assert_allclose(l1, l2, rtol=0, atol=1e-14)


def test_bidir_invariant_under_key_permutation(oracle_mod):
    q, k, v, cu_q, cu_kv = _problem(6, ctx=[12], block=[4])
    perm = np.random.default_rng(0).permutation(k.shape[0])
    o1, l1 = oracle_mod.block_attention(q, k, v, cu_q, cu_kv, 2, BIDIR)
    o2, l2 = oracle_mod.block_attention(q, k[perm], v[perm], cu_q, cu_kv, 2, BIDIR)
    np.testing.assert_allclose(o1, o2, rtol=0, atol=1e-13)
    np.testing.assert_allclose(l1, l2, rtol=0, atol=1e-13)


def test_constant_values_give_constant_output(oracle_mod):
    q, k, v, cu_q, cu_kv = _problem(7, ctx=[10, 4], block=[3, 3])
    c = np.linspace(-1.0, 2.0, v.shape[2])
    v[:] = c
    for mask in (CAUSAL, BIDIR):
        o, _ = oracle_mod.block_attention(q, k, v, cu_q, cu_kv, 2, mask)
        np.testing.assert_allclose(o, np.broadcast_to(c, o.shape), rtol=0, atol=1e-13)


def test_default_scale_is_inverse_sqrt_head_dim(oracle_mod):
    q, k, v, cu_q, cu_kv = _problem(8, ctx=[5], block=[2], d=64)
    o1, _ = oracle_mod.block_attention(q, k, v, cu_q, cu_kv, 2, CAUSAL)
    o2, _ = oracle_mod.block_attention(q, k, v, cu_q, cu_kv, 2, CAUSAL, scale=0.125)
    np.testing.assert_array_equal(o1, o2)


def test_empty_block_and_rejected_arguments(oracle_mod):
    q, k, v, cu_q, cu_kv = _problem(9, ctx=[5, 6], block=[0, 2])
    o, _ = oracle_mod.block_attention(q, k, v, cu_q, cu_kv, 2, CAUSAL)
    assert o.shape[0] == 2
    with pytest.raises(ValueError):
        oracle_mod.block_attention(q, k, v, cu_q, cu_kv, 3, CAUSAL)  # 4 % 3 != 0
