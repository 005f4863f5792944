"""Shared helpers of the GPU parity tests: moving generator scenes to the
device, oracle parameters matching the library's, and the parity checks
(tolerances stated here, used everywhere)."""
import numpy as np
import torch

import paper_2608_13226_gb300 as cp
from paper_2608_13226_gb300 import scenes

# Parity bars (see the design notes): cost entries relative to max(|C|, floor)
COST_RTOL = {"f32": 1e-5, "bf16": 1e-3}
COST_FLOOR = 0.1
# capacity relative to max(v, 1/N)
CAP_RTOL = {"f32": 1e-5, "bf16": 1e-4}
NEAR_TIE = 1e-5      # relative gain gap under which two picks are both correct
OBJ_RTOL = 1e-4      # final coverage objective


def scene(name, seed=0, **override):
    cfg = scenes.config(name, **override) if override else scenes.CONFIGS[name]
    return scenes.make_scene(cfg, seed)


def to_dev(s, device="cuda"):
    f = torch.from_numpy(s["feats"])
    f = f.to(torch.bfloat16) if s["dtype"] == "bf16" else f
    return (f.to(device).contiguous(), torch.from_numpy(s["pos"]).to(device).contiguous(),
            torch.from_numpy(s["frame"]).to(device).contiguous())


def batch_to_dev(scs, device="cuda"):
    parts = [to_dev(s, device) for s in scs]
    return tuple(torch.stack([p[i] for p in parts]).contiguous() for i in range(3))


def oracle_params(orc, p: cp.Params):
    w = orc.Weights(p.lambda_f, p.lambda_x, p.lambda_tau, p.kappa, p.alpha_f, p.alpha_x,
                    p.alpha_tau)
    return orc.Params(weights=w, n_cap=p.n_cap, g=p.g, capacity_mode=p.capacity_mode,
                      m0=p.m0, voxel=p.voxel_m, norm_mode=p.norm_mode)


def assert_cost_close(Cg, Co, dtype, what="cost"):
    Cg = np.asarray(Cg, dtype=np.float64)
    err = np.abs(Cg - Co) / np.maximum(np.abs(Co), COST_FLOOR)
    worst = float(err.max()) if err.size else 0.0
    at = np.unravel_index(int(err.argmax()), err.shape) if err.size else None
    assert worst <= COST_RTOL[dtype], f"{what}: max rel err {worst:.3g} at {at}"
    return worst


def assert_capacity_close(vg, vo, dtype):
    vg = np.asarray(vg, dtype=np.float64)
    N = vo.shape[-1]
    err = np.abs(vg - vo) / np.maximum(np.abs(vo), 1.0 / N)
    worst = float(err.max())
    assert worst <= CAP_RTOL[dtype], f"capacity: max rel err {worst:.3g}"
    return worst


def check_sgs_teacher_forced(orc, C64, v64, order, gains, objective, M0, g=0, nbr=None):
    """Re-run the oracle's greedy on the GPU's own cost and capacity, forced
    to the GPU's picks: every pick must be the oracle's argmax or within
    NEAR_TIE of it, the recorded gains must match, and the objective too."""
    K = len(order)
    res = orc.sgs(C64, v64, K, M0, g, nbr, forced=np.asarray(order, dtype=np.int64))
    diverged = 0
    for l in range(K):
        best = res["best_gain"][l]
        if order[l] != res["best_idx"][l]:
            diverged += 1
            assert best - res["picked_gain"][l] <= NEAR_TIE * best, (
                f"step {l}: GPU picked {order[l]} (gain {res['picked_gain'][l]:.9g}), "
                f"oracle best {res['best_idx'][l]} (gain {best:.9g})")
        assert abs(gains[l] - res["picked_gain"][l]) <= NEAR_TIE * best + 1e-9, (
            f"step {l}: gain {gains[l]:.9g} vs {res['picked_gain'][l]:.9g}")
    assert abs(objective - res["F"]) <= OBJ_RTOL * abs(res["F"]) + 1e-12
    return diverged, res


def _coverage_after(Cm, order, steps, M0, g=0, nbr=None):
    """m_j after the first `steps` picks of `order`: min(M0, min over those
    picks s with j in M_g(s) of C(s, j)) (the coverage cost of the greedy's
    state, by its definition)."""
    N = Cm.shape[0]
    m = np.full(N, float(M0))
    for s in order[:steps]:
        if g and g < N:
            cols = np.concatenate([[s], nbr[s, :g - 1]]).astype(np.int64)
            m[cols] = np.minimum(m[cols], Cm[s, cols])
        else:
            np.minimum(m, Cm[s], out=m)
    return m


def gain_error_bound(Cm, v, m, t, eps, g=0, nbr=None):
    """(gain(t), bound on |gain_gpu(t) - gain(t)|) at coverage state m, when
    every cost entry of the GPU is within eps_c of the oracle's, every
    capacity within eps_v of the oracle's relative to itself (eps = (eps_c,
    eps_v)), and both have picked the same tokens so far (so each m_j is
    within eps_c too).  A term v_j max(m_j - C(t, j), 0) can change only
    where m_j - C(t, j) > -2 eps_c, by at most 2 eps_c v (1 + eps_v) through
    the cost and eps_v of itself through the capacity; the fp32 terms and
    their sum add at most (n + 2) 2^-24 of the gain over n such terms."""
    eps_c, eps_v = eps
    N = Cm.shape[0]
    cols = (np.concatenate([[t], nbr[t, :g - 1]]).astype(np.int64) if g and g < N
            else np.arange(N))
    d = m[cols] - Cm[t, cols]
    gain = float(v[cols] @ np.maximum(d, 0.0))
    near = d > -2.0 * eps_c
    n = int(near.sum())
    return gain, (2.0 * eps_c * (1.0 + eps_v) * float(v[cols][near].sum()) +
                  (eps_v + (n + 2) * 2.0 ** -24) * gain)


def check_sgs_end_to_end(orc, ora, order, kept, M0, g=0, eps=None):
    """GPU (own cost) vs oracle (own cost): identical picks up to the first
    step where the two may legitimately differ, and the final objective (the
    oracle's F on the oracle's cost for both kept sets) within OBJ_RTOL.

    The picks may first differ at a step whose oracle best/second gap is
    below NEAR_TIE relative; or, given eps = (the largest difference between
    the GPU's and the oracle's cost entries, the largest relative difference
    of their capacities), both measured on these inputs, at a
    step where the oracle's gain of its own pick exceeds its gain of the
    GPU's pick by no more than the two gains' error bounds
    (gain_error_bound): the GPU's cost, within eps of the oracle's, cannot
    then decide between them.  Late in a long greedy the gains are 1e-4 of
    the first ones, where a cost rounding of 1e-6 moves a gain by more than
    1e-5 of itself.  Returns (equal steps, Jaccard overlap)."""
    K = len(order)
    first = next((l for l in range(K) if order[l] != ora["order"][l]), K)
    if first < K:
        best, sec = ora["best_gain"][first], ora["second"][first]
        if not best - sec < NEAR_TIE * best:
            assert eps is not None, (
                f"diverged at step {first} without a near-tie: best {best:.9g} second {sec:.9g}")
            nb = ora["nbr"] if ora["g"] < ora["C"].shape[0] else None
            m = _coverage_after(ora["C"], ora["order"], first, M0, ora["g"], nb)
            ga, ea = gain_error_bound(ora["C"], ora["v"], m, int(ora["order"][first]), eps,
                                      ora["g"], nb)
            gb, eb = gain_error_bound(ora["C"], ora["v"], m, int(order[first]), eps, ora["g"], nb)
            assert abs(ga - best) <= 1e-12 * best + 1e-300
            assert ga - gb <= ea + eb, (
                f"diverged at step {first}: oracle gain of its pick {ga:.9g}, of the GPU's pick "
                f"{gb:.9g}; gap {ga - gb:.3g} exceeds the cost-error bound {ea + eb:.3g}")
    nb = ora["nbr"] if ora["g"] < ora["C"].shape[0] else None
    F_gpu_set = orc.objective(ora["C"], ora["v"], kept, M0, ora["g"], nb)
    assert abs(F_gpu_set - ora["F"]) <= OBJ_RTOL * abs(ora["F"]) + 1e-12, (
        f"objective {F_gpu_set:.9g} vs oracle {ora['F']:.9g}")
    jac = len(set(kept.tolist()) & set(ora["kept"].tolist())) / len(set(kept.tolist()) |
                                                                     set(ora["kept"].tolist()))
    return first, jac


def lite_scores(orc, s, w, nm, v, protos, members):
    """Oracle Lite score sum_{j in G} v_j C(t, j) of token protos[i] for the
    group members[i] (oracle arithmetic; v and normalisers as given)."""
    F = s["feats"].astype(np.float64)
    S = np.concatenate([np.full(len(m), t, dtype=np.int64) for t, m in zip(protos, members)])
    T = np.concatenate([np.asarray(m, dtype=np.int64) for m in members])
    c = orc.cost_pairs(F, s["pos"], s["frame"], w, nm, S, T)
    out, at = [], 0
    for m in members:
        out.append(float(c[at:at + len(m)] @ np.asarray(v, dtype=np.float64)[m]))
        at += len(m)
    return np.array(out)


def check_lite_end_to_end(orc, s, ora, kept, group_start, w, dtype="bf16"):
    """GPU Lite (its own normalisers, capacity and groups) against the
    oracle's Lite on the same scene (the oracle's own normalisers, capacity
    and groups; ``ora`` = oracle.lite(...)).

    - Group starts equal the oracle's, except where the oracle's running
      mass lies within 2 CAP_RTOL of the boundary's threshold q/K of the
      total at every position between the two starts: if every capacity is
      within CAP_RTOL of the oracle's, so is every running sum, and a start
      can move only across positions that close to the threshold.
    - Every GPU group holds exactly one kept token.  Where a group is the
      oracle's group, its prototype is the oracle's or within NEAR_TIE of
      the oracle's best score; where a start moved, the prototype of each
      of the two groups it bounds minimises (up to NEAR_TIE) the oracle's
      score over the GPU's members, by brute force.
    - Over the groups both sides share, the oracle's Lite objective of the
      GPU's prototypes is within OBJ_RTOL of the oracle's own (a moved
      start changes the two groups' members, and so their scores, by the
      capacity of the tokens it moves).
    Returns (moved group starts, near-tie prototypes)."""
    kept = np.asarray(kept, dtype=np.int64)
    bg = np.asarray(group_start, dtype=np.int64)
    bo, perm, Q = ora["b"], ora["perm"], ora["Q"]
    K, N = len(kept), len(perm)
    assert bg[0] == 0 and bg[K] == N and np.all(np.diff(bg) >= 1)
    P = np.cumsum(Q.astype(np.float64)[perm])  # running mass in Morton order
    S = P[-1]
    moved = np.flatnonzero(bg != bo)
    for q in moved:
        lo, hi = min(bg[q], bo[q]), max(bg[q], bo[q])
        rel = np.abs(P[lo - 1:hi - 1] * K / (q * S) - 1.0)
        assert rel.max() <= 2 * CAP_RTOL[dtype], (
            f"group {q} starts at {bg[q]} (oracle {bo[q]}), {rel.max():.3g} from the threshold")
    group_of = np.empty(N, dtype=np.int64)
    for q in range(K):
        group_of[perm[bg[q]:bg[q + 1]]] = q
    assert sorted(group_of[kept].tolist()) == list(range(K)), "one prototype per group"
    proto_g = np.empty(K, dtype=np.int64)
    proto_g[group_of[kept]] = kept
    nm, v = ora["norms"], ora["v"]
    members = [perm[bg[q]:bg[q + 1]] for q in range(K)]
    same = (bg[:-1] == bo[:-1]) & (bg[1:] == bo[1:])
    differ = [q for q in range(K) if same[q] and proto_g[q] != ora["proto"][q]]
    if differ:
        sc = lite_scores(orc, s, w, nm, v, proto_g[differ], [members[q] for q in differ])
        for q, x in zip(differ, sc):
            best = ora["score"][q]
            assert x - best <= NEAR_TIE * max(best, 1e-12), (q, proto_g[q], ora["proto"][q], x, best)
    for q in np.flatnonzero(~same):  # the groups a moved start bounds
        mem = members[q]
        sc = lite_scores(orc, s, w, nm, v, mem, [mem] * len(mem))
        x = sc[list(mem).index(proto_g[q])]
        assert x - sc.min() <= NEAR_TIE * max(sc.min(), 1e-12), (q, proto_g[q], x, sc.min())
    shared = np.flatnonzero(same)
    obj = float(lite_scores(orc, s, w, nm, v, proto_g[shared], [members[q] for q in shared]).sum())
    obj_o = float(np.asarray(ora["score"])[shared].sum())
    assert abs(obj - obj_o) <= OBJ_RTOL * abs(obj_o) + 1e-12, (
        f"Lite objective over the {len(shared)} shared groups {obj:.9g} vs oracle {obj_o:.9g}")
    return len(moved), len(differ)


def check_lite_teacher_forced(orc, s, kept, group_start, vg, nm_g, w, voxel):
    """GPU Lite against the oracle's Lite steps run on the GPU's own
    capacity and normalisers: groups bit-exact (integer arithmetic on the
    same fp32 capacities), and every group's prototype the oracle's argmin
    or within NEAR_TIE of its score.  Returns the near-tie count."""
    _, perm = orc.morton(s["pos"], voxel)
    K = len(kept)
    b, _ = orc.lite_groups(vg, perm, K)
    np.testing.assert_array_equal(np.asarray(group_start), b)
    F = s["feats"].astype(np.float64)
    v64 = np.asarray(vg, dtype=np.float64)
    proto, score, _ = orc.lite_select(F, s["pos"], s["frame"], w, nm_g, v64, perm, b)
    group_of = np.empty(len(perm), dtype=np.int64)
    for q in range(K):
        group_of[perm[b[q]:b[q + 1]]] = q
    kept = np.asarray(kept, dtype=np.int64)
    assert sorted(group_of[kept].tolist()) == list(range(K)), "one prototype per group"
    proto_g = np.empty(K, dtype=np.int64)
    proto_g[group_of[kept]] = kept
    differ = np.flatnonzero(proto_g != proto)
    if len(differ):
        sc = lite_scores(orc, s, w, nm_g, v64, proto_g[differ],
                         [perm[b[q]:b[q + 1]] for q in differ])
        for q, x in zip(differ, sc):
            assert x - score[q] <= NEAR_TIE * max(score[q], 1e-12), (q, x, score[q])
    return len(differ)


def measured_errors(Cg, Co, vg, vo):
    """(largest |C_gpu - C_oracle|, largest |v_gpu - v_oracle| / v_oracle)."""
    eps_c = float(np.abs(np.asarray(Cg, dtype=np.float64) - Co).max())
    vo = np.asarray(vo, dtype=np.float64)
    eps_v = float((np.abs(np.asarray(vg, dtype=np.float64) - vo) / np.maximum(vo, 1e-300)).max())
    return eps_c, eps_v
