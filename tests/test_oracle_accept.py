"""Pins for the oracle's lossless speculative acceptance (CPU only).

What fixes the oracle from outside itself:
  * Losslessness (Section 1; Section 3.1 Metrics: the target's output distribution is
    preserved): with drafts sampled from q, the first emitted token is distributed as the
    target distribution p_0, and the token at position i, given that i drafts were
    accepted, as p_i -- chi-square over 10^6 seeded trials on a 16-token vocabulary.
  * The prefix-survival identity of Appendix A.1: with fixed rows, the expected accepted
    length is sum_{i=1}^{gamma} prod_{j<=i} alpha_j, alpha_j = sum_x min(p_j, q_j) (the
    per-position acceptance probability of the ratio test).
  * The geometric form of Appendix A.2 at the paper's own tau = 5.92 (Table 2): rows with
    a common overlap rho give rho (1 - rho^gamma) / (1 - rho).
  * Limits and special cases: T -> 0 reduces to the greedy longest-matching-argmax prefix,
    q = p accepts every draft, disjoint supports accept none and resample inside supp(p),
    E_{x~q}[a(x)] = sum_x min(p, q), and the inverse-CDF sampler reproduces p on a fine
    grid of uniforms.
A swapped ratio (q/p), a residual of the wrong sign, an off-by-one in the prefix, a
missing temperature or a sampler that is not index-ordered fails at least one of these.
"""
import os

import numpy as np
import pytest
from scipy import special, stats

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_tau.txt")


def _golden():
    vals = {}
    with open(GOLDEN) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                name, val = line.split()[:2]
                vals[name] = float(val)
    return vals


def _probs(rng, n, V, conc=2.0):
    return rng.dirichlet(np.full(V, conc), size=n)


def _run_trials(oracle_mod, p_rows, q_rows, n_trials, seed, T=1.0, chunk=125_000):
    """Fixed per-position target rows p_rows [gamma+1, V] and draft rows q_rows [gamma, V] (probabilities);
    drafts sampled from q, logits = T * log(prob) so that softmax(logits / T) = prob."""
    gamma, V = q_rows.shape
    with np.errstate(divide="ignore"):
        tl = T * np.log(p_rows)
        dl = T * np.log(q_rows)
    rng = np.random.default_rng(seed)
    n_acc_all, out_all = [], []
    done = 0
    while done < n_trials:
        n = min(chunk, n_trials - done)
        cdf = np.cumsum(q_rows, axis=1)
        uu = rng.random((n, gamma))
        toks = np.stack([np.minimum(np.searchsorted(cdf[i], uu[:, i], side="right"), V - 1)
                         for i in range(gamma)], axis=1).astype(np.int32)
        target = np.tile(tl, (n, 1))
        draft = np.tile(dl, (n, 1))
        cu = (np.arange(n + 1) * gamma).astype(np.int32)
        res = oracle_mod.spec_accept(target, draft, toks.reshape(-1), cu, T, rng.random(n * gamma), rng.random(n))
        n_acc_all.append(res["n_accepted"])
        out_all.append(res["out_tokens"].reshape(n, gamma + 1))
        done += n
    return np.concatenate(n_acc_all), np.concatenate(out_all)


def _chi2_ok(samples, p, n_min=1000):
    V = len(p)
    counts = np.bincount(samples, minlength=V)
    n = counts.sum()
    assert n >= n_min
    exp = n * p
    stat = ((counts - exp) ** 2 / exp).sum()
    crit = stats.chi2.ppf(1 - 1e-3, V - 1)  # 37.70 at 15 dof
    return stat, crit


@pytest.mark.slow
@pytest.mark.parametrize("T", [1.0, 0.5])
def test_lossless_chi_square_and_prefix_survival(oracle_mod, T):
    V, gamma = 16, 3
    rng = np.random.default_rng(123)
    p_rows = _probs(rng, gamma + 1, V)
    q_rows = _probs(rng, gamma, V)
    n_acc, out = _run_trials(oracle_mod, p_rows, q_rows, 1_000_000, seed=7, T=T)
    # first emitted token ~ p_0
    stat, crit = _chi2_ok(out[:, 0], p_rows[0])
    assert stat < crit, (stat, crit)
    # token at position 1 given one accepted draft ~ p_1
    sel = n_acc >= 1
    stat, crit = _chi2_ok(out[sel, 1], p_rows[1])
    assert stat < crit, (stat, crit)
    # Appendix A.1: E[n_acc] = sum_i prod_{j<=i} alpha_j
    alpha = np.minimum(p_rows[:gamma], q_rows).sum(axis=1)
    expect = np.cumprod(alpha).sum()
    sigma = n_acc.std() / np.sqrt(len(n_acc))
    assert abs(n_acc.mean() - expect) < 5 * sigma, (n_acc.mean(), expect, sigma)


def test_geometric_form_at_paper_tau(oracle_mod):
    """Appendix A.2: equal overlap rho at every position gives rho(1-rho^gamma)/(1-rho); planted at the
    paper's tau = 5.92 (Table 2) with gamma = 15 drafts of a B = 16 block."""
    g = _golden()
    tau, gamma = g["tau_qwen3_4b_t1"], int(g["train_block"]) - 1
    f = lambda r: r * (1 - r ** gamma) / (1 - r) - tau  # noqa: E731
    lo, hi = 0.5, 0.999
    for _ in range(200):
        mid = 0.5 * (lo + hi)
        lo, hi = (mid, hi) if f(mid) < 0 else (lo, mid)
    rho = 0.5 * (lo + hi)
    V = 8
    p = np.array([rho / 2, rho / 2, (1 - rho) / 2, (1 - rho) / 2, 0, 0, 0, 0])
    q = np.array([rho / 2, rho / 2, 0, 0, (1 - rho) / 2, (1 - rho) / 2, 0, 0])
    assert abs(np.minimum(p, q).sum() - rho) < 1e-15
    n_acc, out = _run_trials(oracle_mod, np.tile(p, (gamma + 1, 1)), np.tile(q, (gamma, 1)), 200_000, seed=11)
    sigma = n_acc.std() / np.sqrt(len(n_acc))
    assert abs(n_acc.mean() - tau) < 5 * sigma, (n_acc.mean(), tau, sigma)
    # every emitted token lies in supp(p)
    emitted = out[np.arange(len(out)), n_acc]
    assert np.all(p[emitted] > 0)


def test_greedy_is_longest_matching_argmax_prefix(oracle_mod):
    rng = np.random.default_rng(5)
    V, S = 50, 40
    gammas = rng.integers(0, 7, size=S)
    cu = np.concatenate([[0], np.cumsum(gammas)]).astype(np.int32)
    target = np.round(rng.standard_normal((cu[-1] + S, V)) * 2, 1)  # rounding plants exact ties
    amax = np.argmax(target, axis=1)  # first maximal index
    toks = np.zeros(cu[-1], dtype=np.int32)
    for s in range(S):
        for i in range(gammas[s]):
            t = amax[cu[s] + s + i]
            toks[cu[s] + i] = t if rng.random() < 0.8 else (t + 1) % V
    res = oracle_mod.spec_accept(target, None, toks, cu, 0.0)
    for s in range(S):
        k = 0
        while k < gammas[s] and toks[cu[s] + k] == amax[cu[s] + s + k]:
            k += 1
        assert res["n_accepted"][s] == k
        row = res["out_tokens"][cu[s] + s: cu[s + 1] + s + 1]
        np.testing.assert_array_equal(row[:k], toks[cu[s]:cu[s] + k])
        assert row[k] == amax[cu[s] + s + k]
        assert np.all(row[k + 1:] == -1)
        np.testing.assert_array_equal(res["accept_prob"][cu[s]:cu[s + 1]],
                                      (toks[cu[s]:cu[s + 1]] == amax[cu[s] + s + np.arange(gammas[s])]))


def test_small_temperature_reduces_to_greedy(oracle_mod):
    rng = np.random.default_rng(9)
    V, S, gamma = 200, 30, 6
    cu = (np.arange(S + 1) * gamma).astype(np.int32)
    target = rng.standard_normal((S * (gamma + 1), V)) * 3
    draft = target[np.repeat(np.arange(S), gamma) + np.arange(S * gamma)] + rng.standard_normal((S * gamma, V)) * 0.3
    toks = np.argmax(draft, axis=1).astype(np.int32)
    g0 = oracle_mod.spec_accept(target, None, toks, cu, 0.0)
    g1 = oracle_mod.spec_accept(target, draft, toks, cu, 1e-4, rng.random(S * gamma), rng.random(S))
    # a sequence is a near-tie when a top-2 logit gap of any of its rows is within 50 T
    gap = lambda a: np.diff(np.sort(a, axis=1)[:, -2:], axis=1)[:, 0]  # noqa: E731
    tgap, dgap = gap(target).reshape(S, gamma + 1), gap(draft).reshape(S, gamma)
    clean = (tgap.min(axis=1) > 50 * 1e-4) & (dgap.min(axis=1) > 50 * 1e-4)
    assert clean.sum() >= 0.8 * S
    np.testing.assert_array_equal(g0["n_accepted"][clean], g1["n_accepted"][clean])
    out0, out1 = g0["out_tokens"].reshape(S, gamma + 1), g1["out_tokens"].reshape(S, gamma + 1)
    np.testing.assert_array_equal(out0[clean], out1[clean])
    assert np.any(g0["n_accepted"] > 0) and np.any(g0["n_accepted"] < gamma)


def test_identical_rows_accept_everything(oracle_mod):
    rng = np.random.default_rng(3)
    V, S, gamma = 64, 500, 5
    cu = (np.arange(S + 1) * gamma).astype(np.int32)
    row = rng.standard_normal(V) * 2
    target = np.tile(row, (S * (gamma + 1), 1))
    draft = np.tile(row, (S * gamma, 1))
    toks = rng.integers(0, V, size=S * gamma).astype(np.int32)
    res = oracle_mod.spec_accept(target, draft, toks, cu, 1.0, rng.random(S * gamma), rng.random(S))
    assert np.all(res["accept_prob"] == 1.0)
    assert np.all(res["n_accepted"] == gamma)
    # bonus token ~ p_gamma
    bonus = res["out_tokens"].reshape(S, gamma + 1)[:, gamma]
    assert np.all((bonus >= 0) & (bonus < V))


def test_disjoint_supports_accept_nothing(oracle_mod):
    V, gamma, S = 10, 4, 20_000
    p = np.array([0.1, 0.2, 0.3, 0.4, 0, 0, 0, 0, 0, 0])
    q = np.array([0, 0, 0, 0, 0.25, 0.25, 0.25, 0.25, 0, 0])
    n_acc, out = _run_trials(oracle_mod, np.tile(p, (gamma + 1, 1)), np.tile(q, (gamma, 1)), S, seed=4)
    assert np.all(n_acc == 0)
    counts = np.bincount(out[:, 0], minlength=V)
    assert counts[4:].sum() == 0
    exp = S * p[:4]
    assert ((counts[:4] - exp) ** 2 / exp).sum() < stats.chi2.ppf(1 - 1e-3, 3)


def test_expected_acceptance_over_draft_equals_overlap(oracle_mod):
    rng = np.random.default_rng(21)
    V = 40
    tl = rng.standard_normal(V) * 2
    dl = tl + rng.standard_normal(V)
    for T in (1.0, 0.7, 2.5):
        toks = np.arange(V, dtype=np.int32)
        cu = np.arange(V + 1, dtype=np.int32)  # one drafted token per sequence
        target = np.tile(tl, (2 * V, 1))
        draft = np.tile(dl, (V, 1))
        res = oracle_mod.spec_accept(target, draft, toks, cu, T, np.zeros(V), np.zeros(V))
        p, q = special.softmax(tl / T), special.softmax(dl / T)
        assert abs((q * res["accept_prob"]).sum() - np.minimum(p, q).sum()) < 1e-13
        assert np.all((res["accept_prob"] >= 0) & (res["accept_prob"] <= 1))
        # u = 0 accepts every draft with a > 0
        assert np.all(res["n_accepted"] == (res["accept_prob"] > 0))


def test_inverse_cdf_reproduces_target_on_uniform_grid(oracle_mod):
    """Bonus draw (all drafts accepted): token(u) over a fine grid of u reproduces p_gamma's masses."""
    rng = np.random.default_rng(8)
    V, n = 12, 120_000
    tl = rng.standard_normal(V)
    p = special.softmax(tl)
    u = (np.arange(n) + 0.5) / n
    target = np.tile(tl, (n, 1))
    res = oracle_mod.spec_accept(target, np.zeros((0, V)), np.zeros(0, np.int32), np.zeros(n + 1, np.int32), 1.0,
                                 np.zeros(0), u)
    frac = np.bincount(res["out_tokens"], minlength=V) / n
    np.testing.assert_allclose(frac, p, atol=2.0 / n)
    # index order: tokens are non-decreasing in u
    assert np.all(np.diff(res["out_tokens"]) >= 0)


def test_residual_draw_matches_normalised_positive_part(oracle_mod):
    """At a rejection the emitted token follows max(0, p - q) / Z (grid over the sampling uniform)."""
    rng = np.random.default_rng(12)
    V, n = 9, 90_000
    tl, dl = rng.standard_normal(V) * 2, rng.standard_normal(V) * 2
    p, q = special.softmax(tl), special.softmax(dl)
    r = np.maximum(p - q, 0)
    r /= r.sum()
    x0 = int(np.argmax(q / p))  # a draft with a < 1
    target = np.tile(tl, (2 * n, 1))
    draft = np.tile(dl, (n, 1))
    res = oracle_mod.spec_accept(target, draft, np.full(n, x0, np.int32), np.arange(n + 1, dtype=np.int32), 1.0,
                                 np.full(n, 0.999999), (np.arange(n) + 0.5) / n)
    assert np.all(res["n_accepted"] == 0)
    frac = np.bincount(res["out_tokens"].reshape(n, 2)[:, 0], minlength=V) / n
    np.testing.assert_allclose(frac, r, atol=2.0 / n)


def test_margins_are_reported(oracle_mod):
    rng = np.random.default_rng(2)
    V, S, gamma = 100, 50, 4
    cu = (np.arange(S + 1) * gamma).astype(np.int32)
    target = rng.standard_normal((S * (gamma + 1), V))
    draft = rng.standard_normal((S * gamma, V))
    toks = rng.integers(0, V, S * gamma).astype(np.int32)
    ua = rng.random(S * gamma)
    res = oracle_mod.spec_accept(target, draft, toks, cu, 1.0, ua, rng.random(S))
    for s in range(S):
        k = res["n_accepted"][s]
        upto = min(k + 1, gamma)
        m = np.abs(ua[s * gamma:s * gamma + upto] - res["accept_prob"][s * gamma:s * gamma + upto]).min()
        assert res["ratio_margin"][s] == m
        assert 0 <= res["cdf_margin"][s] <= 1


def test_rejects_bad_arguments(oracle_mod):
    with pytest.raises(ValueError):
        oracle_mod.spec_accept(np.zeros((2, 4)), np.zeros((1, 4)), np.array([4], np.int32), [0, 1], 1.0,
                               np.zeros(1), np.zeros(1))  # token id >= V
    with pytest.raises(ValueError):
        oracle_mod.spec_accept(np.zeros((2, 4)), None, np.array([0], np.int32), [0, 1], 1.0, np.zeros(1),
                               np.zeros(1))  # T > 0 needs draft logits
