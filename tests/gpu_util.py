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


def check_sgs_end_to_end(orc, ora, order, kept, M0, g=0):
    """GPU (own cost) vs oracle (own cost): identical picks up to the first
    oracle near-tie; final objective (oracle's F on the oracle's cost for both
    kept sets) within OBJ_RTOL."""
    K = len(order)
    first = next((l for l in range(K) if order[l] != ora["order"][l]), K)
    if first < K:
        best, sec = ora["best_gain"][first], ora["second"][first]
        assert best - sec < NEAR_TIE * best, (
            f"diverged at step {first} without a near-tie: best {best:.9g} second {sec:.9g}")
    nb = ora["nbr"] if ora["g"] < ora["C"].shape[0] else None
    F_gpu_set = orc.objective(ora["C"], ora["v"], kept, M0, ora["g"], nb)
    assert abs(F_gpu_set - ora["F"]) <= OBJ_RTOL * abs(ora["F"]) + 1e-12, (
        f"objective {F_gpu_set:.9g} vs oracle {ora['F']:.9g}")
    jac = len(set(kept.tolist()) & set(ora["kept"].tolist())) / len(set(kept.tolist()) |
                                                                     set(ora["kept"].tolist()))
    return first, jac
