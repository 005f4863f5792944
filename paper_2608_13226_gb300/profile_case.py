"""Run one CoverPrune entry point on a seeded synthetic workload, for
profilers (ncu) and quick timing.

    python -m paper_2608_13226_gb300.profile_case --scene long_video --op select \
        [--batch B] [--K K] [--g G] [--norm-mode M] [--sgs-mode S] [--warmup W] [--repeat R]
        [--stages]

Prints one JSON line with the median CUDA-event time of the call.
"""
from __future__ import annotations

import argparse
import json
import statistics

import numpy as np
import torch

from . import binding as cp
from . import scenes


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--scene", default="long_video", choices=sorted(scenes.CONFIGS))
    ap.add_argument("--op", default="select", choices=("select", "lite", "cost"))
    ap.add_argument("--batch", type=int, default=1)
    ap.add_argument("--N", type=int, default=0, help="override the scene's token count")
    ap.add_argument("--K", type=int, default=0, help="0 = the workload's budget")
    ap.add_argument("--g", type=int, default=0)
    ap.add_argument("--norm-mode", type=int, default=0, choices=(0, 1),
                    help="feature normaliser: 0 min-max over all pairs, 1 bounded (d_f / 2)")
    ap.add_argument("--sgs-mode", type=int, default=0, choices=(0, 1, 2),
                    help="0 lazy, 1 every gain every step, 2 the rule as printed (entropic OT)")
    ap.add_argument("--warmup", type=int, default=1)
    ap.add_argument("--repeat", type=int, default=3)
    ap.add_argument("--stages", action="store_true",
                    help="also report the per-stage split of the timed calls")
    a = ap.parse_args()
    cfg = scenes.config(a.scene, N=a.N) if a.N else scenes.CONFIGS[a.scene]
    sc = [scenes.make_scene(cfg, seed) for seed in range(a.batch)]
    feats = np.stack([s["feats"] for s in sc])
    f = torch.from_numpy(feats)
    f = (f.to(torch.bfloat16) if cfg.dtype == "bf16" else f).cuda()
    pos = torch.from_numpy(np.stack([s["pos"] for s in sc])).cuda()
    fr = torch.from_numpy(np.stack([s["frame"] for s in sc])).cuda()
    K = a.K or cfg.K
    prm = cp.Params(g=a.g, norm_mode=a.norm_mode, sgs_mode=a.sgs_mode)
    if a.op == "select":
        ws = cp.workspace(cp.CP_OP_SELECT, a.batch, cfg.N, cfg.D, K, cp._dtype(f), prm)
        run = lambda: cp.coverprune_select(f, pos, fr, K, prm, ws=ws)
    elif a.op == "lite":
        ws = cp.workspace(cp.CP_OP_LITE, a.batch, cfg.N, cfg.D, K, cp._dtype(f), prm)
        run = lambda: cp.coverprune_lite_select(f, pos, fr, K, prm, ws=ws)
    else:
        ws = cp.workspace(cp.CP_OP_COST, a.batch, cfg.N, cfg.D, 0, cp._dtype(f), prm)
        out = {"cost": torch.empty(a.batch, cfg.N, cfg.N, device="cuda")}
        run = lambda: cp.coverprune_cost(f, pos, fr, prm, ws=ws, out=out)
    for _ in range(a.warmup):
        run()
    torch.cuda.synchronize()
    if a.stages:
        cp.coverprune_profile_read()
        cp.coverprune_profile_enable(True)
    times = []
    for _ in range(a.repeat):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        run()
        e1.record()
        torch.cuda.synchronize()
        times.append(e0.elapsed_time(e1))
    stages = None
    if a.stages:
        cp.coverprune_profile_enable(False)
        stages = {k: round(v[0] / a.repeat, 3) for k, v in cp.coverprune_profile_read().items()
                  if v[0] > 0}
    st = cp.coverprune_check(ws)
    line = {"scene": a.scene, "op": a.op, "batch": a.batch, "N": cfg.N, "D": cfg.D, "K": K,
            "g": a.g, "ms_median": statistics.median(times), "status": cp.status_string(st)}
    if stages is not None:
        line["stages_ms"] = stages
    if a.op == "select":
        line["call_stats"] = cp.coverprune_call_stats(ws)
    print(json.dumps(line))
    if st != cp.CP_OK:
        raise SystemExit(1)


if __name__ == "__main__":
    main()
