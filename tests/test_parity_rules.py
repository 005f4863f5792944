"""The parity rules of the GPU tests, checked on the CPU with the oracle
alone: a run on a cost perturbed within eps (standing in for the GPU's
rounded cost) passes the end-to-end rule, and a planted wrong pick fails
it."""
import numpy as np
import pytest

from gpu_util import NEAR_TIE, check_sgs_end_to_end, measured_errors


def _scene(orc, seed, N=300, D=16):
    rng = np.random.default_rng(seed)
    modes = rng.normal(size=(6, D))
    F = modes[rng.integers(6, size=N)] + 0.5 * rng.normal(size=(N, D))
    X = (rng.random((N, 3)) * 4.0).astype(np.float32)
    tau = np.sort(rng.integers(4, size=N)).astype(np.int32)
    prm = orc.Params()
    return F, X, tau, prm


@pytest.mark.parametrize("seed", [0, 2, 3, 4])
def test_perturbed_cost_passes_end_to_end(orc, seed):
    """A greedy run on the oracle's cost perturbed by up to eps = 2e-5 first
    picks differently from the oracle's at a step whose best/second gap is
    above the 1e-5 near-tie bar (late in the run, where gains are 1e-3 of
    the first ones); the cost-error bound accepts it, and the objectives
    agree within 1e-4."""
    F, X, tau, prm = _scene(orc, seed, N=500)
    K = 300
    ora = orc.select(F, X, tau, K, prm)
    rng = np.random.default_rng(50 + seed)
    eps_c = 2e-5
    Cp = ora["C"] + rng.uniform(-eps_c, eps_c, ora["C"].shape)
    np.fill_diagonal(Cp, 0.0)
    vp = ora["v"] * (1.0 + rng.uniform(-1e-7, 1e-7, ora["v"].shape))
    gpu = orc.sgs(Cp, vp, K, prm.M0())
    first = next(l for l in range(K) if gpu["order"][l] != ora["order"][l])
    assert ora["best_gain"][first] - ora["second"][first] >= NEAR_TIE * ora["best_gain"][first]
    eps = measured_errors(Cp, ora["C"], vp, ora["v"])
    assert check_sgs_end_to_end(orc, ora, gpu["order"], gpu["kept"], prm.M0(), eps=eps)[0] == first
    with pytest.raises(AssertionError):  # without the measured errors: only the near-tie bar
        check_sgs_end_to_end(orc, ora, gpu["order"], gpu["kept"], prm.M0())


def test_wrong_pick_fails_end_to_end(orc):
    F, X, tau, prm = _scene(orc, 7)
    K = 40
    ora = orc.select(F, X, tau, K, prm)
    # plant a mistake: at the step with the largest relative best/second gap,
    # take the oracle's second choice instead of its best
    gaps = (ora["best_gain"] - ora["second"]) / ora["best_gain"]
    l = int(np.argmax(gaps[:-1]))
    assert gaps[l] > 1e-3
    # the runner-up at step l: the best candidate other than the oracle's pick
    alt = None
    for t in range(ora["C"].shape[0]):
        if t in set(ora["order"][:l + 1].tolist()):
            continue
        trial = np.concatenate([ora["order"][:l], [t]])
        r = orc.sgs(ora["C"], ora["v"], l + 1, prm.M0(), forced=trial)
        if abs(r["picked_gain"][l] - ora["second"][l]) <= 1e-12 * ora["best_gain"][l]:
            alt = t
            break
    assert alt is not None
    bad = np.concatenate([ora["order"][:l], [alt]])
    rest = [t for t in ora["order"][l:] if t != alt][:K - l - 1]
    bad = np.concatenate([bad, rest]).astype(np.int64)
    assert len(set(bad.tolist())) == K
    with pytest.raises(AssertionError):
        check_sgs_end_to_end(orc, ora, bad, np.sort(bad), prm.M0(), eps=(1e-7, 1e-7))
