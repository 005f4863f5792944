"""Pins of the oracle's literal SGS (Sec. 3.5 as printed: Eqs.
srpot_sinkhorn, greedy_flow, sgs_select, sgs_update) and of its entropic
semi-relaxed OT solver, against what the mathematics fixes:

- the one-source problem in closed form (water-filling: P_j = min(v_j,
  lambda exp(-C_j / eps)) with the total mass fixed, lambda by bisection);
- the optimality conditions of the entropic problem (row marginals equal u,
  column sums at most v, and equal to v wherever the column potential is
  below 0);
- the limit eps -> 0 against the linear program of Eq. srpot (scipy), within
  the entropic gap eps M log(m N) of a plan of mass M over m x N entries;
- hand-derived selections: the first pick is the capacity-weighted medoid
  (the coverage-gain greedy's first pick), identical tokens and g = 1 give
  the lowest indices, and two far clusters show where the residual rule
  picks its second token.
The GPU's literal mode is compared with this oracle in the GPU tests; the
paper fixes neither eps nor the iteration count, so the rule itself is
parity-unpinned beyond these cases."""
import math

import numpy as np
import pytest
from scipy.optimize import linprog


def _rand_problem(seed, m, N):
    rng = np.random.default_rng(seed)
    C = rng.random((m, N)) * 2.0
    v = rng.random(N) + 0.1
    v /= v.sum()
    u = np.full(m, 1.0 / (m + 2))
    return C, u, v


def _water_fill(c, v, mass, eps):
    """min(v_j, lam exp(-c_j / eps)) summing to mass, lam by bisection on log lam."""
    lo, hi = -200.0, 200.0
    for _ in range(300):
        mid = 0.5 * (lo + hi)
        s = np.minimum(v, np.exp(mid - c / eps)).sum()
        lo, hi = (mid, hi) if s < mass else (lo, mid)
    return np.minimum(v, np.exp(0.5 * (lo + hi) - c / eps))


@pytest.mark.parametrize("eps", [0.5, 0.05, 0.01])
def test_one_source_water_filling(orc, eps):
    rng = np.random.default_rng(3)
    N = 9
    c = rng.random(N)
    v = rng.random(N) + 0.05
    v /= v.sum()
    mass = 0.4
    res = orc.sot_sinkhorn(c[None, :], [mass], v, eps, 400)
    np.testing.assert_allclose(res["P"][0], _water_fill(c, v, mass, eps), rtol=1e-9, atol=1e-14)


@pytest.mark.parametrize("seed", range(3))
def test_marginals_and_slackness(orc, seed):
    C, u, v = _rand_problem(seed, 4, 11)
    eps = 0.1
    res = orc.sot_sinkhorn(C, u, v, eps, 3000)
    P, g = res["P"], res["g"]
    np.testing.assert_allclose(P.sum(1), u, rtol=1e-10)
    col = P.sum(0)
    np.testing.assert_allclose(res["colsum"], col, rtol=1e-12)
    assert np.all(col <= v * (1 + 1e-12))
    assert np.all(g <= 0.0)
    tight = g < -1e-9
    assert tight.any()
    np.testing.assert_allclose(col[tight], v[tight], rtol=1e-9)
    # the plan has the Gibbs form of the dual potentials
    np.testing.assert_allclose(P, np.exp((res["f"][:, None] + g[None, :] - C) / eps), rtol=1e-12)


def _sot_lp(C, u, v):
    m, N = C.shape
    A_eq = np.zeros((m, m * N))
    for i in range(m):
        A_eq[i, i * N:(i + 1) * N] = 1.0
    A_ub = np.zeros((N, m * N))
    for j in range(N):
        A_ub[j, j::N] = 1.0
    r = linprog(C.ravel(), A_ub=A_ub, b_ub=v, A_eq=A_eq, b_eq=u, bounds=(0, None),
                method="highs")
    assert r.status == 0
    return r.fun


@pytest.mark.parametrize("seed", range(3))
def test_small_eps_approaches_the_lp(orc, seed):
    C, u, v = _rand_problem(10 + seed, 3, 8)
    lp = _sot_lp(C, u, v)
    M = u.sum()
    gaps = []
    for eps in (0.2, 0.05, 0.01):
        res = orc.sot_sinkhorn(C, u, v, eps, 200000)
        P = res["P"]
        np.testing.assert_allclose(P.sum(1), u, rtol=1e-8)
        assert np.all(P.sum(0) <= v * (1 + 1e-12))
        gap = float((C * P).sum()) - lp
        assert -1e-9 <= gap <= eps * M * math.log(C.size) + 1e-9, (eps, gap)
        gaps.append(gap)
    assert gaps[-1] < gaps[0]


def _scene(orc, seed, N=40):
    rng = np.random.default_rng(seed)
    F = rng.normal(size=(N, 5)) + rng.integers(0, 3, N)[:, None]
    X = (rng.random((N, 3)) * 3).astype(np.float32)
    tau = np.sort(rng.integers(0, 4, N)).astype(np.int32)
    w = orc.Weights()
    nm = orc.normalisers(F, X, tau)
    Cm = orc.cost_matrix(F, X, tau, w, nm)
    _, v = orc.capacity(F, X, tau, w, nm, 3)
    return Cm, v, X


@pytest.mark.parametrize("seed", range(4))
def test_first_pick_is_the_weighted_medoid(orc, seed):
    Cm, v, _ = _scene(orc, seed)
    lit = orc.sgs_literal(Cm, v, 1, 0.05, 10)
    gain = orc.sgs(Cm, v, 1, 3.0)  # the coverage-gain greedy's first pick
    assert lit["order"][0] == gain["order"][0]
    assert lit["best_score"][0] == pytest.approx(float(Cm[lit["order"][0]] @ v), rel=1e-12)


def test_identical_tokens_and_single_token_neighbourhoods(orc):
    N, K = 12, 5
    Cz = np.zeros((N, N))
    v = np.full(N, 1.0 / N)
    assert orc.sgs_literal(Cz, v, K, 0.05, 20)["order"].tolist() == list(range(K))
    Cm, v2, X = _scene(orc, 7, N=N)
    np.fill_diagonal(Cm, 0.0)  # C(t, t) = 0 exactly (the fp64 cost rounds 1 - cos to ~1e-16)
    nbr = orc.knn_others(X, 2)
    # g = 1: M_g(t) = {t}, every score r_t C(t, t) = 0 -> lowest indices
    assert orc.sgs_literal(Cm, v2, K, 0.05, 20, g=1, nbr_g=nbr)["order"].tolist() == \
        list(range(K))


@pytest.mark.parametrize("a,second_in", [(0.6, "B"), (0.8, "A")])
def test_two_far_clusters(orc, a, second_in):
    """Clusters A (tokens 0..4, mass a) and B (tokens 5..9, mass 1 - a),
    cost 0 inside a cluster and 1 across; K = 2, so each source carries 1/2.
    Step 0 picks the lowest index of the heavier cluster A (score 1 - a
    against a).  Step 1: the plan sends the source's 1/2 into A at no cost
    (up to exp(-1/eps)), leaving residual a - 1/2 in A and 1 - a in B; a
    token of A scores 1 - a, one of B a - 1/2, so the second pick is token 5
    when a < 3/4 and token 1 when a > 3/4."""
    N = 10
    lab = np.array([0] * 5 + [1] * 5)
    Cm = (lab[:, None] != lab[None, :]).astype(np.float64)
    v = np.where(lab == 0, a / 5, (1 - a) / 5)
    res = orc.sgs_literal(Cm, v, 2, 0.02, 200)
    assert res["order"][0] == 0
    assert res["order"][1] == (5 if second_in == "B" else 1)
    want = (a - 0.5) if second_in == "B" else (1 - a)
    assert res["best_score"][1] == pytest.approx(want, abs=1e-9)


@pytest.mark.parametrize("seed", range(3))
def test_residual_mass_and_forcing(orc, seed):
    Cm, v, _ = _scene(orc, 20 + seed)
    K = 6
    own = orc.sgs_literal(Cm, v, K, 0.05, 40)
    again = orc.sgs_literal(Cm, v, K, 0.05, 40, forced=own["order"])
    for k in ("order", "best_idx", "best_score", "second", "picked_score"):
        np.testing.assert_array_equal(own[k], again[k], err_msg=k)
    # after the last step's plan, the residual holds the untransported mass
    # 1 - l / K (row marginals exact after convergence, columns capped)
    l = K - 1
    res = orc.sot_sinkhorn(Cm[own["order"][:l]], np.full(l, 1.0 / K), v, 0.05, 5000)
    r = np.maximum(v - res["colsum"], 0.0)
    assert r.sum() == pytest.approx(1.0 - l / K, rel=1e-9)
    forced = np.random.default_rng(seed).permutation(Cm.shape[0])[:K]
    f = orc.sgs_literal(Cm, v, K, 0.05, 40, forced=forced)
    np.testing.assert_array_equal(f["order"], forced)
    assert np.all(f["picked_score"] >= f["best_score"])
    with pytest.raises(ValueError):
        orc.sgs_literal(Cm, v, 2, 0.05, 40, forced=np.array([3, 3]))
