"""Pins of the CPU oracle against what the paper and the mathematics fix.

None of these tests retypes the oracle's formulas: each checks the oracle
against a hand-worked closed form (tests/golden/worked_example.json), an
exhaustive search, a linear program solved by scipy (the OT problems of
Eqs. srpot and blk_ot themselves), a library routine (scipy KD-tree, pdist,
numpy matmul) or an invariant that a dropped term, a wrong sign, a wrong index
or a transposed operand would break.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
from scipy.optimize import linprog
from scipy.spatial import cKDTree
from scipy.spatial.distance import pdist

HERE = os.path.dirname(os.path.abspath(__file__))
GOLD = json.load(open(os.path.join(HERE, "golden", "worked_example.json")))


def ev(expr: str) -> float:
    """Evaluate a hand-derived closed form (log and rationals only)."""
    return float(eval(expr, {"__builtins__": {}}, {"log": math.log}))


def ex_inputs():
    F = np.array(GOLD["features"], dtype=np.float64)
    X = np.array(GOLD["positions"], dtype=np.float32)
    tau = np.array(GOLD["frames"], dtype=np.int32)
    return F, X, tau


def rand_scene(rng, N, D=6, frames=3, box=2.0, n_modes=3):
    modes = rng.normal(size=(n_modes, D))
    lab = rng.integers(n_modes, size=N)
    F = modes[lab] + 0.4 * rng.normal(size=(N, D))
    X = (rng.random((N, 3)) * box).astype(np.float32)
    tau = np.sort(rng.integers(frames, size=N)).astype(np.int32)
    return F, X, tau


# --------------------------------------------------------------------------
# Worked example (Eqs. fst_metrics, fst_cost, fst_capacity_score,
# fst_capacity, SGS, Lite)
# --------------------------------------------------------------------------

def test_worked_example_norms_and_cost(orc):
    F, X, tau = ex_inputs()
    nm = orc.normalisers(F, X, tau)
    for k, e in GOLD["norms"].items():
        assert getattr(nm, k) == pytest.approx(ev(e), abs=1e-12), k
    Cm = orc.cost_matrix(F, X, tau, orc.Weights(kappa=GOLD["kappa"]), nm)
    want = np.array([[ev(e) for e in row] for row in GOLD["cost"]])
    np.testing.assert_allclose(Cm, want, atol=1e-12, rtol=0)


def test_worked_example_bounded_normaliser(orc):
    """The bounded feature normaliser (d_f / 2) on the worked example: hand
    values of the norms, the cost matrix and the uniform SGS."""
    F, X, tau = ex_inputs()
    bn = GOLD["bounded_norm"]
    nm = orc.normalisers(F, X, tau, norm_mode=1)
    for k, e in bn["norms"].items():
        assert getattr(nm, k) == pytest.approx(ev(e), abs=1e-12), k
    Cm = orc.cost_matrix(F, X, tau, orc.Weights(kappa=GOLD["kappa"]), nm)
    want = np.array([[ev(e) for e in row] for row in bn["cost"]])
    np.testing.assert_allclose(Cm, want, atol=1e-12, rtol=0)
    v = np.full(3, 1.0 / 3.0)
    M0 = GOLD["M0"]
    for t, e in enumerate(bn["uniform_step1_gains"]):
        assert M0 - orc.objective(Cm, v, [t], M0) == pytest.approx(ev(e), abs=1e-12)
    res = orc.sgs(Cm, v, 2, M0)
    assert list(res["order"]) == bn["uniform_K2_order"]
    after = bn["uniform_step2_gains_after_1"]
    assert res["best_gain"][1] == pytest.approx(ev(after["2"]), abs=1e-12)
    assert res["second"][1] == pytest.approx(ev(after["0"]), abs=1e-12)
    assert res["F"] == pytest.approx(ev(bn["uniform_K2_F"]), abs=1e-12)
    # end to end through the driver's parameter
    prm = orc.Params(weights=orc.Weights(kappa=GOLD["kappa"]), capacity_mode=1, m0=M0,
                     norm_mode=1)
    r = orc.select(F, X, tau, 2, prm)
    assert list(r["order"]) == bn["uniform_K2_order"]


def test_bounded_normaliser_equals_minmax_with_antipodal_pair(orc):
    """A scene holding f and -f has min cos = -1, so the measured feature
    range is [0, 2] and both normalisers give the same cost; the spatial and
    temporal ranges never depend on the mode."""
    rng = np.random.default_rng(11)
    F, X, tau = rand_scene(rng, 40)
    F[7] = -F[3]
    a = orc.normalisers(F, X, tau, norm_mode=0)
    b = orc.normalisers(F, X, tau, norm_mode=1)
    assert a.f_lo == pytest.approx(0.0, abs=1e-12) and a.f_hi == pytest.approx(2.0, abs=1e-12)
    assert (a.x_lo, a.x_hi, a.tau_lo, a.tau_hi) == (b.x_lo, b.x_hi, b.tau_lo, b.tau_hi)
    w = orc.Weights()
    np.testing.assert_allclose(orc.cost_matrix(F, X, tau, w, a), orc.cost_matrix(F, X, tau, w, b),
                               atol=1e-12, rtol=0)
    # without the antipodal pair the feature term is scaled by range / 2
    F2, X2, tau2 = rand_scene(np.random.default_rng(12), 40)
    a2 = orc.normalisers(F2, X2, tau2, norm_mode=0)
    b2 = orc.normalisers(F2, X2, tau2, norm_mode=1)
    assert a2.f_hi < 2.0 and (b2.f_lo, b2.f_hi) == (0.0, 2.0)
    wf = orc.Weights(lambda_x=0.0, lambda_tau=0.0)
    Ca = orc.cost_matrix(F2, X2, tau2, wf, a2)
    Cb = orc.cost_matrix(F2, X2, tau2, wf, b2)
    np.testing.assert_allclose(Cb, Ca * (a2.f_hi - a2.f_lo) / 2.0, atol=1e-12, rtol=0)


def test_worked_example_uniform_sgs(orc):
    F, X, tau = ex_inputs()
    w = orc.Weights(kappa=GOLD["kappa"])
    nm = orc.normalisers(F, X, tau)
    Cm = orc.cost_matrix(F, X, tau, w, nm)
    u = GOLD["uniform"]
    v = np.array([ev(e) for e in u["v"]])
    M0 = GOLD["M0"]
    # step-1 gains of every candidate = F(empty) - F({t})
    F0 = M0 * v.sum()
    for t, e in enumerate(u["step1_gains"]):
        assert F0 - orc.objective(Cm, v, [t], M0) == pytest.approx(ev(e), abs=1e-12)
    res = orc.sgs(Cm, v, 2, M0)
    assert list(res["order"]) == u["K2_order"]
    assert list(res["kept"]) == u["K2_kept"]
    assert res["best_gain"][0] == pytest.approx(ev(u["step1_gains"][1]), abs=1e-12)
    assert res["best_gain"][1] == pytest.approx(ev(u["step2_gains_after_1"]["2"]), abs=1e-12)
    assert res["second"][1] == pytest.approx(ev(u["step2_gains_after_1"]["0"]), abs=1e-12)
    assert res["F"] == pytest.approx(ev(u["K2_F"]), abs=1e-12)


def test_worked_example_capacity_and_fst_sgs(orc):
    F, X, tau = ex_inputs()
    w = orc.Weights(kappa=GOLD["kappa"])
    nm = orc.normalisers(F, X, tau)
    fc = GOLD["fst_capacity_n1"]
    nbr = orc.knn_others(X, 1)
    assert nbr.tolist() == fc["nbr"]  # token 1: equidistant 0 and 2 -> lower index
    r, v = orc.capacity(F, X, tau, w, nm, 1)
    np.testing.assert_allclose(r, [ev(e) for e in fc["r"]], atol=1e-12)
    np.testing.assert_allclose(v, [ev(e) for e in fc["v"]], atol=1e-12)
    Cm = orc.cost_matrix(F, X, tau, w, nm)
    res = orc.sgs(Cm, v, 2, GOLD["M0"])
    assert res["order"][0] == fc["K2_first"]
    assert res["best_gain"][0] == pytest.approx(ev(fc["step1_gains"][2]), abs=1e-12)
    assert res["second"][0] == pytest.approx(ev(fc["step1_gains"][1]), abs=1e-12)
    # step 2 is an exact tie between tokens 0 and 1: both have gain 5/7
    assert res["best_gain"][1] == pytest.approx(5 / 7, abs=1e-12)
    assert res["second"][1] == pytest.approx(5 / 7, abs=1e-12)
    assert res["order"][1] in (0, 1)
    assert res["F"] == pytest.approx(ev(fc["K2_F"]), abs=1e-12)


def test_worked_example_lite(orc):
    F, X, tau = ex_inputs()
    lk = GOLD["lite_K2_voxel0.2"]
    codes, perm = orc.morton(X, 0.2)
    assert codes.tolist() == lk["codes"]
    assert perm.tolist() == lk["perm"]
    for mode in (0, 1):
        prm = orc.Params(weights=orc.Weights(kappa=GOLD["kappa"]), n_cap=1,
                         capacity_mode=mode, voxel=0.2)
        res = orc.lite(F, X, tau, 2, prm)
        assert res["b"].tolist() == lk["b"]
        assert res["kept"].tolist() == lk["kept"]


# --------------------------------------------------------------------------
# The objective is the OT value of Eq. srpot (source capacity free) and the
# Lite objective is the value of Eq. blk_ot: both solved as LPs by scipy.
# --------------------------------------------------------------------------

def sot_lp(Cm, v, S, M0=None, allowed=None):
    """min <C, P> s.t. P >= 0 supported on rows S, P^T 1 = v (sum u = 1 with
    u free), optionally restricted to allowed[s, j] with an extra source of
    cost M0 that may serve anyone."""
    N = Cm.shape[0]
    rows = list(S)
    costs, A = [], []
    cols = []
    for si, s in enumerate(rows):
        for j in range(N):
            if allowed is None or allowed[s, j]:
                costs.append(Cm[s, j])
                cols.append(j)
    if M0 is not None:
        for j in range(N):
            costs.append(M0)
            cols.append(j)
    A = np.zeros((N, len(costs)))
    for c, j in enumerate(cols):
        A[j, c] = 1.0
    out = linprog(np.array(costs), A_eq=A, b_eq=v, bounds=(0, None), method="highs")
    assert out.status == 0
    return out.fun


@pytest.mark.parametrize("seed", range(4))
def test_objective_is_semi_relaxed_ot_value(orc, seed):
    rng = np.random.default_rng(100 + seed)
    N = 9
    F, X, tau = rand_scene(rng, N)
    w = orc.Weights()
    nm = orc.normalisers(F, X, tau)
    Cm = orc.cost_matrix(F, X, tau, w, nm)
    _, v = orc.capacity(F, X, tau, w, nm, 3)
    M0 = 3.0
    for S in ([0], [2, 5], [1, 4, 7, 8]):
        assert orc.objective(Cm, v, S, M0) == pytest.approx(sot_lp(Cm, v, S), abs=1e-9)
    # local neighbourhoods M_g: transport only inside M_g(s), unserved mass at M0
    g = 4
    nbr = orc.knn_others(X, g - 1)
    allowed = np.zeros((N, N), dtype=bool)
    for s in range(N):
        allowed[s, s] = True
        allowed[s, nbr[s]] = True
    for S in ([0], [2, 5], [1, 4, 7]):
        assert orc.objective(Cm, v, S, M0, g, nbr) == pytest.approx(
            sot_lp(Cm, v, S, M0, allowed), abs=1e-9)


@pytest.mark.parametrize("seed", range(3))
def test_lite_objective_is_block_ot_value(orc, seed):
    """Eqs. blk_plan / blk_ot: with group masses exactly 1/K the block LP's
    value for the chosen prototypes equals the Lite objective, and the Lite
    prototypes minimise it over all choices (brute force)."""
    rng = np.random.default_rng(200 + seed)
    N, K = 12, 3
    F, X, tau = rand_scene(rng, N)
    w = orc.Weights()
    nm = orc.normalisers(F, X, tau)
    Cm = orc.cost_matrix(F, X, tau, w, nm)
    v = np.full(N, 1.0 / N)  # N/K tokens per group -> mass exactly 1/K
    _, perm = orc.morton(X, 0.2)
    b, _ = orc.lite_groups(v, perm, K)
    assert np.all(np.diff(b) == N // K)
    proto, score, obj = orc.lite_select(F, X, tau, w, nm, v, perm, b)
    groups = [perm[b[q]:b[q + 1]] for q in range(K)]

    def block_lp(protos):
        costs, cols, rows = [], [], []
        for q, s in enumerate(protos):
            for j in groups[q]:
                costs.append(Cm[s, j]); cols.append(j); rows.append(q)
        A = np.zeros((N + K, len(costs)))
        for c, (j, q) in enumerate(zip(cols, rows)):
            A[j, c] = 1.0
            A[N + q, c] = 1.0
        beq = np.concatenate([v, np.full(K, 1.0 / K)])
        out = linprog(np.array(costs), A_eq=A, b_eq=beq, bounds=(0, None), method="highs")
        assert out.status == 0
        return out.fun

    assert obj == pytest.approx(block_lp(proto), abs=1e-9)
    best = min(block_lp(c) for c in itertools.product(*groups))
    assert obj == pytest.approx(best, abs=1e-9)
    for q in range(K):
        brute = min(groups[q], key=lambda t: (sum(v[j] * Cm[t, j] for j in groups[q]), t))
        assert proto[q] == brute


# --------------------------------------------------------------------------
# Exhaustive search on tiny scenes: greedy properties (Sec. 3.5, submodular
# guarantee)
# --------------------------------------------------------------------------

@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("g", [0, 3])
def test_greedy_exhaustive(orc, seed, g):
    rng = np.random.default_rng(seed)
    N = int(rng.integers(7, 11))
    K = int(rng.integers(2, 5))
    F, X, tau = rand_scene(rng, N)
    w = orc.Weights()
    nm = orc.normalisers(F, X, tau)
    Cm = orc.cost_matrix(F, X, tau, w, nm)
    _, v = orc.capacity(F, X, tau, w, nm, 2)
    M0 = 3.0
    nbr = orc.knn_others(X, g - 1) if g else None
    res = orc.sgs(Cm, v, K, M0, g, nbr)
    obj = lambda S: orc.objective(Cm, v, S, M0, g, nbr)
    # first pick = best singleton (lowest index on ties)
    singles = [obj([t]) for t in range(N)]
    assert res["order"][0] == int(np.argmin(singles))
    # the recorded gain is the exact decrease of the objective
    prev = M0 * v.sum()
    for l in range(K):
        cur = obj(res["order"][:l + 1])
        assert cur == pytest.approx(res["F_after"][l], abs=1e-12)
        assert prev - cur == pytest.approx(res["picked_gain"][l], abs=1e-12)
        assert cur <= prev + 1e-15
        prev = cur
    assert np.all(np.diff(res["best_gain"]) <= 1e-12)  # diminishing returns
    # (1 - 1/e) guarantee of greedy for monotone submodular maximisation
    opt = min(obj(list(S)) for S in itertools.combinations(range(N), K))
    f0 = M0 * v.sum()
    assert f0 - res["F"] >= (1 - 1 / math.e) * (f0 - opt) - 1e-12
    assert len(set(res["order"].tolist())) == K


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("g", [0, 3])
def test_greedy_forced_order(orc, seed, g):
    """Teacher forcing (the GPU parity tests drive the oracle's greedy along
    the GPU's picks): forcing the oracle's own order reproduces its unforced
    run exactly; forcing any other legal order adds exactly those tokens,
    records as picked gain the exact objective decrease of each forced
    addition, and still reports at every step the brute-force best addition
    (argmax of the decrease over the unselected tokens, lowest index on
    ties) and the runner-up's decrease."""
    rng = np.random.default_rng(100 + seed)
    N = int(rng.integers(7, 11))
    K = int(rng.integers(2, 6))
    F, X, tau = rand_scene(rng, N)
    w = orc.Weights()
    nm = orc.normalisers(F, X, tau)
    Cm = orc.cost_matrix(F, X, tau, w, nm)
    _, v = orc.capacity(F, X, tau, w, nm, 2)
    M0 = 3.0
    nbr = orc.knn_others(X, g - 1) if g else None
    own = orc.sgs(Cm, v, K, M0, g, nbr)
    again = orc.sgs(Cm, v, K, M0, g, nbr, forced=own["order"])
    for k in ("order", "best_idx", "best_gain", "second", "picked_gain", "F_after"):
        np.testing.assert_array_equal(again[k], own[k], err_msg=k)
    np.testing.assert_array_equal(own["order"], own["best_idx"])
    obj = lambda S: orc.objective(Cm, v, S, M0, g, nbr)
    for trial in range(3):
        forced = rng.permutation(N)[:K]
        res = orc.sgs(Cm, v, K, M0, g, nbr, forced=forced)
        np.testing.assert_array_equal(res["order"], forced)
        prev = M0 * v.sum()
        for l in range(K):
            S = list(forced[:l])
            dec = np.array([prev - obj(S + [t]) if t not in S else -np.inf for t in range(N)])
            best = int(np.argmax(dec))  # first maximum = lowest index on exact ties
            assert res["best_idx"][l] == best
            assert res["best_gain"][l] == pytest.approx(dec[best], abs=1e-12)
            rest = np.delete(dec, best)
            second = rest.max() if np.isfinite(rest).any() else -1.0
            assert res["second"][l] == pytest.approx(second, abs=1e-12)
            cur = obj(S + [int(forced[l])])
            assert res["picked_gain"][l] == pytest.approx(prev - cur, abs=1e-12)
            assert res["F_after"][l] == pytest.approx(cur, abs=1e-12)
            prev = cur
    # a repeated or out-of-range forced token is an error, not a silent pick
    with pytest.raises(ValueError):
        orc.sgs(Cm, v, 2, M0, g, nbr, forced=np.array([1, 1]))
    with pytest.raises(ValueError):
        orc.sgs(Cm, v, 1, M0, g, nbr, forced=np.array([N]))


# --------------------------------------------------------------------------
# Closed forms
# --------------------------------------------------------------------------

@pytest.mark.parametrize("g", [0, 4])
def test_identical_tokens(orc, g):
    N, K = 13, 5
    F = np.tile(np.array([[0.3, -1.2, 0.7, 2.0]]), (N, 1))
    X = np.tile(np.array([[1.0, 2.0, 0.5]], dtype=np.float32), (N, 1))
    tau = np.zeros(N, dtype=np.int32)
    prm = orc.Params(g=g)
    res = orc.select(F, X, tau, K, prm)
    np.testing.assert_allclose(res["C"], 0.0, atol=1e-12)
    np.testing.assert_allclose(res["v"], 1.0 / N, atol=1e-15)
    if g == 0:
        assert res["kept"].tolist() == list(range(K))
        assert res["F"] == pytest.approx(0.0, abs=1e-12)
    else:
        # token 0 covers {0..g-1}; afterwards only tokens >= g still have an
        # uncovered neighbourhood member (themselves), lowest index first
        assert res["kept"].tolist() == [0] + list(range(g, g + K - 1))
        # the N - (g + K - 1) tokens nobody covers keep m = M0
        assert res["F"] == pytest.approx(3.0 * (N - g - K + 1) / N, abs=1e-12)
    lt = orc.lite(F, X, tau, K, prm)
    assert lt["kept"].tolist() == [math.ceil(q * N / K) for q in range(K)]
    assert lt["objective"] == pytest.approx(0.0, abs=1e-12)


@pytest.mark.parametrize("seed", range(3))
def test_k1_weighted_medoid_and_lite_agree(orc, seed):
    rng = np.random.default_rng(300 + seed)
    N = 15
    F, X, tau = rand_scene(rng, N)
    prm = orc.Params(n_cap=3)
    res = orc.select(F, X, tau, 1, prm)
    scores = res["C"] @ res["v"]
    assert res["kept"][0] == int(np.argmin(scores))
    lt = orc.lite(F, X, tau, 1, prm)
    assert lt["kept"][0] == res["kept"][0]
    assert lt["objective"] == pytest.approx(scores.min(), abs=1e-12)


@pytest.mark.parametrize("N", [9, 10])
def test_collinear_centre(orc, N):
    F = np.ones((N, 3))
    X = np.zeros((N, 3), dtype=np.float32)
    X[:, 0] = np.arange(N, dtype=np.float32)
    tau = np.zeros(N, dtype=np.int32)
    prm = orc.Params(capacity_mode=1)
    # the centre has the element-wise smallest sorted distance multiset; for
    # even N the two centres tie exactly in real arithmetic, and which one
    # wins then depends only on the rounding of two equal sums
    legal = {(N - 1) // 2} if N % 2 else {N // 2 - 1, N // 2}
    assert orc.select(F, X, tau, 1, prm)["kept"][0] in legal
    assert orc.lite(F, X, tau, 1, prm)["kept"][0] in legal


def test_k_equals_n(orc):
    rng = np.random.default_rng(7)
    N = 11
    F, X, tau = rand_scene(rng, N)
    for g in (0, 3):
        res = orc.select(F, X, tau, N, orc.Params(g=g, n_cap=2))
        assert res["kept"].tolist() == list(range(N))
        assert res["F"] == pytest.approx(0.0, abs=1e-12)
    lt = orc.lite(F, X, tau, N, orc.Params(n_cap=2))
    assert lt["kept"].tolist() == list(range(N))
    assert lt["objective"] == pytest.approx(0.0, abs=1e-12)


def test_temporal_direction(orc):
    """C(s,t) = ReLU(tau_s - tau_t)/M_tau for identical f and x: covering an
    earlier token with a later one costs; K=1 picks the first token of frame 0
    (a transposed ReLU would pick from the last frame)."""
    frames, per = 4, 3
    N = frames * per
    F = np.ones((N, 2))
    X = np.zeros((N, 3), dtype=np.float32)
    tau = np.repeat(np.arange(frames), per).astype(np.int32)
    rng = np.random.default_rng(3)
    p = rng.permutation(N)
    tau = tau[p]
    w = orc.Weights()
    nm = orc.normalisers(F, X, tau)
    Cm = orc.cost_matrix(F, X, tau, w, nm)
    want = np.maximum(tau[:, None] - tau[None, :], 0) / (frames - 1)
    np.testing.assert_allclose(Cm, want, atol=1e-12)
    res = orc.select(F, X, tau, 1, orc.Params(capacity_mode=1))
    assert res["kept"][0] == int(np.flatnonzero(tau == 0).min())


# --------------------------------------------------------------------------
# Invariants of the cost (Eq. fst_cost)
# --------------------------------------------------------------------------

def test_cost_invariants(orc):
    rng = np.random.default_rng(11)
    N = 40
    F, X, tau = rand_scene(rng, N, D=8, frames=5)
    nm = orc.normalisers(F, X, tau)
    w = orc.Weights(lambda_f=0.7, lambda_x=1.3, lambda_tau=0.4, kappa=5.0)
    Cm = orc.cost_matrix(F, X, tau, w, nm)
    np.testing.assert_allclose(np.diag(Cm), 0.0, atol=1e-12)
    # only the temporal term is asymmetric
    dt = (tau[:, None] - tau[None, :]) / (tau.max() - tau.min())
    np.testing.assert_allclose(Cm - Cm.T, w.lambda_tau * dt, atol=1e-12)
    assert Cm.min() >= -1e-12
    assert Cm.max() <= w.lambda_f + w.lambda_x + w.lambda_tau + 1e-12
    # each normalised term reaches exactly 1 somewhere and 0 on the diagonal
    for one in ("lambda_f", "lambda_x", "lambda_tau"):
        kw = {"lambda_f": 0.0, "lambda_x": 0.0, "lambda_tau": 0.0, one: 1.0}
        Cone = orc.cost_matrix(F, X, tau, orc.Weights(**kw), nm)
        assert Cone.max() == pytest.approx(1.0, abs=1e-12)
        assert Cone.min() == pytest.approx(0.0, abs=1e-12)
    # lambda_f = 0 removes every dependence on the features
    w0 = orc.Weights(lambda_f=0.0)
    F2 = rng.normal(size=F.shape)
    nm2 = orc.normalisers(F2, X, tau)
    np.testing.assert_allclose(orc.cost_matrix(F, X, tau, w0, nm),
                               orc.cost_matrix(F2, X, tau, w0, nm2), atol=1e-12)


def test_cost_spatial_term_reduces_to_pdist(orc):
    """kappa -> 0 makes phi_kappa the identity: the spatial-only cost is the
    Euclidean distance matrix (scipy pdist) over its maximum."""
    rng = np.random.default_rng(12)
    N = 30
    F, X, tau = rand_scene(rng, N)
    nm = orc.normalisers(F, X, tau)
    Cm = orc.cost_matrix(F, X, tau, orc.Weights(lambda_f=0, lambda_tau=0, kappa=1e-9), nm)
    from scipy.spatial.distance import squareform
    Dm = squareform(pdist(X.astype(np.float64)))
    np.testing.assert_allclose(Cm, Dm / Dm.max(), atol=1e-8)
    # and kappa large is log-compressed: phi is concave, so phi(x) >= x
    Ck = orc.cost_matrix(F, X, tau, orc.Weights(lambda_f=0, lambda_tau=0, kappa=50.0), nm)
    assert np.all(Ck >= Dm / Dm.max() - 1e-12)
    x = Dm / Dm.max()
    np.testing.assert_allclose(Ck, np.log1p(50 * x) / np.log1p(50), atol=1e-12)


def test_normalisers_match_library_routines(orc):
    rng = np.random.default_rng(13)
    N = 60
    F, X, tau = rand_scene(rng, N, D=16, frames=7)
    F[5] = 0.0  # a zero feature: cos := 0 against everyone, d_f = 1
    nm = orc.normalisers(F, X, tau)
    nrm = np.linalg.norm(F, axis=1)
    G = F @ F.T
    with np.errstate(invalid="ignore", divide="ignore"):
        cos = G / np.outer(nrm, nrm)
    cos[~np.isfinite(cos)] = 0.0
    cos = np.clip(cos, -1, 1)
    assert nm.f_hi == pytest.approx(1 - cos.min(), abs=1e-12)
    assert nm.f_lo == pytest.approx(0.0, abs=1e-12)
    assert nm.x_hi == pytest.approx(pdist(X.astype(np.float64)).max(), abs=1e-12)
    assert nm.x_lo == 0.0 and nm.tau_lo == 0.0
    assert nm.tau_hi == tau.max() - tau.min()


# --------------------------------------------------------------------------
# Neighbours, capacity, Morton, grouping
# --------------------------------------------------------------------------

def test_knn_matches_kdtree(orc):
    rng = np.random.default_rng(14)
    N, k = 300, 9
    X = (rng.random((N, 3)) * 4).astype(np.float32)
    got = orc.knn_others(X, k)
    _, idx = cKDTree(X.astype(np.float64)).query(X.astype(np.float64), k=k + 1)
    for j in range(N):
        want = [i for i in idx[j] if i != j][:k]
        assert got[j].tolist() == want


def test_knn_ties_lower_index_first(orc):
    X = np.zeros((6, 3), dtype=np.float32)
    X[:, 0] = [0, 1, -1, 1, -1, 2]
    got = orc.knn_others(X, 4)
    assert got[0].tolist() == [1, 2, 3, 4]  # all at distance 1
    X2 = np.zeros((4, 3), dtype=np.float32)  # all coincident
    assert orc.knn_others(X2, 3).tolist() == [[1, 2, 3], [0, 2, 3], [0, 1, 3], [0, 1, 2]]


def test_capacity_properties(orc):
    rng = np.random.default_rng(15)
    N = 50
    F, X, tau = rand_scene(rng, N)
    X[17] = np.array([40.0, 40.0, 40.0], dtype=np.float32)  # a far outlier
    w = orc.Weights()
    nm = orc.normalisers(F, X, tau)
    r, v = orc.capacity(F, X, tau, w, nm, 4)
    assert v.sum() == pytest.approx(1.0, abs=1e-12)
    assert np.all(v >= 0)
    assert int(np.argmax(v)) == 17
    np.testing.assert_allclose(v, r / r.sum(), rtol=1e-12)
    _, vu = orc.capacity(F, X, tau, w, nm, 4, mode=1)
    np.testing.assert_allclose(vu, 1.0 / N)
    # n = 0 neighbours: r == 0 everywhere -> uniform fallback
    _, v0 = orc.capacity(F, X, tau, w, nm, 0)
    np.testing.assert_allclose(v0, 1.0 / N)


def test_morton_codes(orc):
    X = np.array([[0, 0, 0], [1, 0, 0], [0, 1, 0], [0, 0, 1], [1, 1, 1], [2, 0, 0],
                  [1023, 0, 0], [5000, 0, 0]], dtype=np.float32)
    codes, perm = orc.morton(X, 1.0)
    q1023 = sum(1 << (3 * i) for i in range(10))
    assert codes.tolist() == [0, 1, 2, 4, 7, 8, q1023, q1023]  # clamped to 1023
    assert perm.tolist() == list(range(8))
    # scrambled input: the permutation sorts by (code, index)
    order = [5, 7, 3, 0, 6, 1, 4, 2]
    codes2, perm2 = orc.morton(X[order], 1.0)
    assert codes2.tolist() == [codes[i] for i in order]
    # old tokens 6 and 7 share the clamped code; in the scrambled input old 7
    # sits at index 1 and old 6 at index 4, so old 7 comes first
    assert [order[i] for i in perm2] == [0, 1, 2, 3, 4, 5, 7, 6]


@pytest.mark.parametrize("N,K", [(12, 3), (12, 4), (20, 5), (7, 7)])
def test_uniform_groups_are_equal_runs(orc, N, K):
    v = np.full(N, 1.0 / N)
    b, _ = orc.lite_groups(v, np.arange(N), K)
    assert b.tolist() == [q * N // K for q in range(K + 1)]


@pytest.mark.parametrize("case", range(5))
def test_groups_adversarial(orc, case):
    rng = np.random.default_rng(case)
    N, K = 30, 6
    if case == 0:
        v = np.zeros(N); v[3] = 0.9; v[4:] = 0.1 / (N - 4)      # one heavy token
    elif case == 1:
        v = np.zeros(N); v[-1] = 1.0                              # all mass at the end
    elif case == 2:
        v = np.zeros(N); v[0] = 1.0                               # all mass first
    elif case == 3:
        v = np.zeros(N)                                           # no mass at all
    else:
        v = rng.pareto(1.0, N); v /= v.sum()
    perm = rng.permutation(N)
    b, _ = orc.lite_groups(v, perm, K)
    assert b[0] == 0 and b[-1] == N and len(b) == K + 1
    assert np.all(np.diff(b) >= 1)


def test_groups_mass_close_to_one_over_k(orc):
    rng = np.random.default_rng(21)
    N, K = 4000, 100
    v = rng.random(N) + 0.5
    v /= v.sum()
    perm = rng.permutation(N)
    b, _ = orc.lite_groups(v, perm, K)
    mass = np.array([v[perm[b[q]:b[q + 1]]].sum() for q in range(K)])
    # each group closes at the first token that reaches its share, so it
    # overshoots 1/K by less than one token's mass
    cum = np.cumsum(mass)
    target = np.arange(1, K + 1) / K
    assert np.all(cum >= target - 1e-9)
    assert np.all(cum - target < v.max() + 1e-9)
