"""GPU parity of bp_tau_select (Appendix A's acceptance-length model) against the fp64 oracle.

Tolerance, derived from the arithmetic: the kernel forms tau = sum_{i<=b} r^i P_i in fp32 with
P_i = prod_{j<=i} gamma_j and r^i as running products (b roundings each), r itself from expf (at most
2 ulp, raised to the i-th power), and b fused multiply-adds of positive terms; the relative error
of tau is at most (5 b + 4) 2^-24.  B* is compared exactly unless the oracle's two best candidates
are within twice that of each other (then either is accepted); regret and the Lipschitz constant
carry the same bound on the tau values they are made of.
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


def rel_tol(bmax: int) -> float:
    return (5 * bmax + 4) * 2.0 ** -24


def run(inp, predicted=True):
    g = to_dev(inp["gamma"])
    cand = inp["candidates"]  # a host array
    pred = to_dev(inp["predicted"]) if predicted else None
    ws = bp.workspace(bp.tau_select_workspace_size(g.shape[0]), dev())
    tau, best, regret, summary = bp.tau_select(g, cand, inp["train_block"], inp["alpha"], predicted=pred, ws=ws)
    status = bp.get_status(ws)
    return (tau.cpu().numpy(), best.cpu().numpy(), None if regret is None else regret.cpu().numpy(),
            summary.cpu().numpy(), status)


def compare(inp, gpu, predicted=True):
    tau, best, regret, summary, status = gpu
    assert status == 0
    ref = oracle.tau_select(inp["gamma"], inp["candidates"], inp["train_block"], inp["alpha"],
                            predicted=inp["predicted"] if predicted else None)
    cand = inp["candidates"]
    tol = rel_tol(int(cand.max()))
    rt = ref["tau"]
    assert np.all(np.abs(tau - rt) <= tol * np.abs(rt) + 1e-30), np.max(np.abs(tau - rt) / np.abs(rt))
    top2 = np.sort(rt, axis=1)[:, -2:] if rt.shape[1] > 1 else np.concatenate([rt, rt - 1], axis=1)
    near = (top2[:, 1] - top2[:, 0]) <= 2 * tol * top2[:, 1]
    assert np.array_equal(best[~near], ref["best"][~near])
    # near-ties: the GPU's choice is one of the two best
    ci = np.searchsorted(cand, best[near])
    assert np.all(rt[near, ci] >= top2[near, 0] * (1 - 2 * tol))
    lips = np.max(np.abs(np.diff(tau, axis=1)) / np.diff(cand)[None, :], axis=1) if len(cand) > 1 else 0
    if predicted:
        pi = np.searchsorted(cand, inp["predicted"])
        tb = np.take_along_axis(tau, np.searchsorted(cand, best)[:, None], axis=1)[:, 0]
        np.testing.assert_allclose(regret, tb - tau[np.arange(len(best)), pi], rtol=0, atol=1e-6)
        assert np.all(np.abs(regret - ref["regret"]) <= 2 * tol * rt.max(axis=1) + 1e-7)
        d = np.abs(best - inp["predicted"])
        assert summary[1] == pytest.approx(d.mean(), rel=1e-12)
        assert abs(summary[0] - ref["summary"][0]) <= 2 * tol * rt.max() + 1e-9
        if not near.any():
            assert summary[1] == ref["summary"][1]
    assert abs(summary[2] - ref["summary"][2]) <= 2 * tol * ref["summary"][2] + 1e-7
    if len(cand) > 1:
        assert summary[2] == pytest.approx(float(np.max(lips)), rel=1e-6)
    return int(near.sum())


@pytest.mark.parametrize("n", [1, 255, 1001, 40000])
def test_default_workload_sizes(n):
    inp = wl.tau_inputs(n, seed=60 + n)
    compare(inp, run(inp))


def test_geometric_form_one_gamma_per_request():
    inp = wl.tau_inputs(5000, seed=70)
    inp["gamma"] = np.ascontiguousarray(inp["gamma"][:, :1])
    compare(inp, run(inp))


def test_other_candidates_and_long_rows():
    inp = wl.tau_inputs(3000, jmax=64, seed=71, train_block=20, alpha=0.003)
    inp["candidates"] = np.array([4, 5, 9, 20, 33, 50, 64], dtype=np.int32)
    rng = np.random.default_rng(72)
    inp["predicted"] = rng.choice(inp["candidates"], size=3000).astype(np.int32)
    compare(inp, run(inp))


def test_without_prediction():
    inp = wl.tau_inputs(3000, seed=73)
    compare(inp, run(inp, predicted=False), predicted=False)


def test_full_size_and_determinism():
    """The benchmark's 4M requests, as bench.py launches it; the summary is bit-identical over calls."""
    inp = wl.tau_inputs(1 << 22)
    first = run(inp)
    compare(inp, first)
    again = run(inp)
    np.testing.assert_array_equal(first[3], again[3])
    np.testing.assert_array_equal(first[1], again[1])


def test_bad_inputs():
    """A predicted size that is no candidate is caught on the device (flag); candidates that do not
    increase, or exceed the rows, are refused on the host."""
    inp = wl.tau_inputs(300, seed=74)
    bad = dict(inp, predicted=inp["predicted"].copy())
    bad["predicted"][7] = 15  # not a candidate
    assert run(bad)[4] == 6
    for cand in ([8, 12, 10], [8, 30]):  # not increasing; longer than the 24-position rows
        with pytest.raises(bp.BlockPilotError):
            run(dict(inp, candidates=np.array(cand, dtype=np.int32)))
