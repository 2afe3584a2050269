"""Pins of the oracle's Appendix A acceptance-length model (tau(b; x), B*(x), regret) against what
the mathematics fixes: exhaustive enumeration of acceptance patterns (the expectation of the
stopping time itself, not the survival formula), the general and geometric forms on constant
predictability, the limits alpha = 0 and gamma = 1, the per-request regret bound, and the
monotonicity of B* in the predictability that Appendix A.2 derives."""
import itertools

import numpy as np
import pytest

import oracle

CAND = np.arange(8, 25, 2, dtype=np.int32)


def enumerate_expected_length(q):
    """E[number of leading accepted drafts] by summing over all 2^b accept/reject patterns, each with
    its probability prod (q_j or 1 - q_j)."""
    b = len(q)
    total = 0.0
    for pattern in itertools.product((0, 1), repeat=b):
        prob = np.prod([qj if a else 1.0 - qj for a, qj in zip(pattern, q)])
        lead = next((i for i, a in enumerate(pattern) if not a), b)
        total += prob * lead
    return total


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_tau_is_the_expected_stopping_time(seed):
    """Appendix A.1: tau is E[L_b]; checked by enumeration with q_j = gamma_j r(b; B)."""
    rng = np.random.default_rng(seed)
    cand = np.array([4, 6, 8, 10], dtype=np.int32)
    gamma = rng.uniform(0.3, 0.99, size=(2, 10))
    B, alpha = 7, 0.05
    res = oracle.tau_select(gamma, cand, B, alpha)
    for x in range(2):
        for c, b in enumerate(cand):
            q = gamma[x, :b] * np.exp(-alpha * (b - B) ** 2)
            assert abs(res["tau"][x, c] - enumerate_expected_length(q)) < 1e-12


def test_geometric_form_equals_the_general_form_on_constant_rows():
    """Appendix A.2: with gamma_j = gamma_x the sum is the finite geometric series (two different
    evaluations in the oracle: the product loop and rho (1 - rho^b) / (1 - rho))."""
    gx = np.array([0.2, 0.5, 0.86, 0.95, 0.999, 1.0])
    general = oracle.tau_select(np.repeat(gx[:, None], 24, axis=1), CAND, 16, 0.002)
    geometric = oracle.tau_select(gx[:, None], CAND, 16, 0.002)
    np.testing.assert_allclose(geometric["tau"], general["tau"], rtol=1e-11)
    np.testing.assert_array_equal(geometric["best"], general["best"])


def test_limits():
    """alpha = 0 and gamma = 1: every draft accepted, tau(b) = b, B* = the largest candidate;
    the retention is 1 at the training size whatever alpha is."""
    res = oracle.tau_select(np.ones((1, 24)), CAND, 16, 0.0)
    np.testing.assert_allclose(res["tau"][0], CAND, rtol=1e-15)
    assert res["best"][0] == 24
    g = np.random.default_rng(3).uniform(0.5, 0.99, size=(1, 24))
    a = oracle.tau_select(g, np.array([16], dtype=np.int32), 16, 0.0)
    b = oracle.tau_select(g, np.array([16], dtype=np.int32), 16, 5.0)
    assert a["tau"][0, 0] == b["tau"][0, 0]


def test_regret_and_its_bound():
    """Appendix A.3: R >= 0, R = 0 at B_hat = B*, R(x) <= L(x) |B* - B_hat|, and the adjacent-pair
    Lipschitz constant equals the one over all candidate pairs."""
    rng = np.random.default_rng(4)
    gx = rng.beta(12, 2, size=500)
    gamma = np.clip(gx[:, None] + rng.normal(0, 0.03, size=(500, 24)), 0.05, 0.999)
    pred = rng.choice(CAND, size=500)
    res = oracle.tau_select(gamma, CAND, 16, 0.001, predicted=pred)
    d = np.abs(res["best"] - pred)
    assert np.all(res["regret"] >= 0)
    assert np.all(res["regret"][d == 0] == 0)
    assert np.all(res["regret"] <= res["lips"] * d + 1e-12)
    t = res["tau"]
    pairs = [(i, j) for i in range(len(CAND)) for j in range(i + 1, len(CAND))]
    full = np.max([np.abs(t[:, i] - t[:, j]) / (CAND[j] - CAND[i]) for i, j in pairs], axis=0)
    np.testing.assert_allclose(res["lips"], full, rtol=1e-12)
    s = res["summary"]
    assert s[0] == pytest.approx(res["regret"].mean()) and s[1] == pytest.approx(d.mean())
    assert s[2] == pytest.approx(res["lips"].max()) and s[3] >= s[0]


def test_optimal_size_grows_with_predictability():
    """Appendix A.2: more predictable samples sustain longer prefixes, so B*(gamma_x) is
    non-decreasing in gamma_x; the retention keeps it near the training size."""
    gx = np.linspace(0.5, 0.999, 200)[:, None]
    best = oracle.tau_select(gx, CAND, 16, 0.001)["best"]
    assert np.all(np.diff(best) >= 0)
    assert best[0] <= 16 <= best[-1]


def test_rejects_bad_candidates():
    with pytest.raises(ValueError):
        oracle.tau_select(np.ones((1, 24)), np.array([8, 8], dtype=np.int32), 16, 0.1)
    with pytest.raises(ValueError):
        oracle.tau_select(np.ones((1, 10)), np.array([8, 12], dtype=np.int32), 16, 0.1)
