#!/usr/bin/env python
"""Throughput benchmark of the GB300 CoverPrune hot path.

Workload (one step): a batch of 32 independent long-video scenes (N=8192
tokens of D=3584 bf16 features, 32 frames x 256 tokens, Zipf-sized modes,
random-walk camera), full CoverPrune at 15% retention (K=1229): FST cost,
FST capacity and dense SGS (every token's neighbourhood is the whole scene),
then the kept indices.  The metric is scenes per second (whole job, all
GPUs; each rank prunes its own 32 scenes -- weak scaling, no collective on
the data path).  The same line reports the dominant kernel's roofline, an
end-to-end number through host buffers, the CPU oracle timed on one whole
scene, and every other workload: the single-scene pruning latency of the
tiny, short-clip, long-video (dense and local) and Lite scenes, and the
32-scene batch at 5/10/15/25% retention for SGS and Lite.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

With --impl reference the CPU oracle (fp64, scalar C) is timed on the host's
cores; each step prunes one whole long-video scene of the workload.
"""
from __future__ import annotations

import argparse
import dataclasses
import datetime
import json
import math
import multiprocessing as mp
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "scenes/sec & pruning latency (N=8192,D=3584,15% keep); % HBM / tensor roofline"
WORKLOAD = "batch32_long_video_full_sgs_15pct"
SCENES, RETENTION = 32, 0.15
SCENE_NAME = "long_video"
LOCAL_G = 64  # local neighbourhood size of the local-SGS measurement
HBM_NOMINAL_GBS = 7900.0  # the part's nominal HBM3e bandwidth, for context beside the measured peak


def _gen(seed):
    """Worker: one scene as bf16 bit patterns (spawned before any CUDA use)."""
    from paper_2608_13226_gb300 import scenes
    s = scenes.make_scene(SCENE_NAME, seed)
    return scenes.bf16_bits(s["feats"]), s["pos"], s["frame"]


def make_batch(seeds):
    procs = max(1, min(len(seeds), (os.cpu_count() or 2) // 2, 16))
    with mp.get_context("spawn").Pool(procs) as pool:
        return pool.map(_gen, seeds)


def rank_seeds(rank: int, per_rank: int = SCENES) -> list:
    """Scene seeds of one rank: every rank prunes its own scenes (weak
    scaling across scenes, no collective on the data path)."""
    return list(range(rank * per_rank, rank * per_rank + per_rank))


def reduce_max(x: float, dist, device) -> float:
    """Max of a per-rank number over all ranks (identity without a process
    group): the whole job lasts as long as its slowest rank."""
    if dist is None:
        return x
    import torch
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(scenes_per_rank: int, world: int, ms_max: float) -> float:
    """Scenes per second of the whole job."""
    return scenes_per_rank * world / (ms_max / 1000.0)


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return d["hbm_gbs"], d["bf16_tflops"], d.get("bf16_tflops_sustained"), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, 1900.0, 1700.0, "fallback"


# --------------------------------------------------------------------------
# clocks under load
# --------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None
        self.window = None  # (start, end) of the timed region, local wall time

    def wait_first_sample(self, limit_s: float = 3.0):
        """Returns once nvidia-smi has written a row (or after limit_s)."""
        t0 = time.time()
        while self.proc is not None and time.time() - t0 < limit_s:
            try:
                if os.path.getsize(self.path) > 0:
                    return
            except OSError:
                return
            time.sleep(0.02)

    def mark(self, start: bool):
        now = datetime.datetime.now()
        self.window = (now, None) if start else (self.window[0] if self.window else now, now)

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-i", str(self.index), "-lms", "50", "-f", self.path],
                stdout=subprocess.DEVNULL, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self) -> dict:
        rows = []
        try:
            for line in open(self.path):
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 10:
                    rows.append(parts)
        except OSError:
            pass
        finally:
            try:
                os.unlink(self.path)
            except OSError:
                pass
        # keep the samples taken inside the timed window (all, if none is)
        inside = []
        if self.window and self.window[1] is not None:
            for r in rows:
                try:
                    t = datetime.datetime.strptime(r[0], "%Y/%m/%d %H:%M:%S.%f")
                except ValueError:
                    continue
                if self.window[0] <= t <= self.window[1]:
                    inside.append(r)
        scope = "timed region" if inside else "whole sampler run"
        rows = inside or rows
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"], "samples": 0}
        sm = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        mx = [float(r[3]) for r in rows if r[3].replace(".", "").isdigit()]
        pw = [float(r[4]) for r in rows if r[4].replace(".", "").isdigit()]
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        reasons = sorted({n for r in rows for n, v in zip(names, r[6:10]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None,
                "power_w_max": max(pw) if pw else None,
                "reasons": reasons, "samples": len(rows), "scope": scope,
                "interval_ms": 50}


# --------------------------------------------------------------------------
# CPU oracle: one whole scene of the workload
# --------------------------------------------------------------------------
def oracle_scene_seconds(scene, K: int) -> tuple[float, dict]:
    """Time the CPU oracle pruning one whole scene of the workload: the
    normalisers over all pairs, capacity neighbours and capacity, the full
    cost matrix and all K greedy steps (the steps oracle.select chains).
    The bf16 features are widened to the oracle's fp64 input before the
    clock starts."""
    import numpy as np

    import oracle as orc
    F = scene["feats"].astype(np.float64)
    X, tau = scene["pos"], scene["frame"]
    prm = orc.Params()
    t0 = time.perf_counter()
    pre = orc.prepare(F, X, tau, prm)
    t1 = time.perf_counter()
    Cm = orc.cost_matrix(F, X, tau, prm.weights, pre["norms"])
    t2 = time.perf_counter()
    orc.sgs(Cm, pre["v"], K, prm.M0())
    t3 = time.perf_counter()
    del Cm
    N, D = F.shape
    sample = (f"one whole {SCENE_NAME} scene (N={N}, D={D}, K={K}): normalisers over all "
              f"pairs, neighbours, capacity, the full cost matrix and all {K} greedy steps")
    parts = {"normalisers_neighbours_capacity": t1 - t0, "cost": t2 - t1, "sgs": t3 - t2}
    return t3 - t0, {"parts_s": {k: round(v_, 3) for k, v_ in parts.items()}, "sample": sample}


def cpu_baseline_line(scene, K):
    import oracle as orc
    orc.build()
    secs, info = oracle_scene_seconds(scene, K)
    return {"value": 1.0 / secs, "unit": "scenes/s", "cores": orc.get_threads(),
            "kind": "oracle", "sample": info["sample"], "scene_s": round(secs, 3),
            "parts_s": info["parts_s"]}


def workload_config(rank: int, B: int, N: int, D: int, K: int) -> dict:
    """The headline workload, identical in both arms' lines."""
    return {"workload": WORKLOAD, "scenes_per_gpu": B, "N": N, "D": D, "K": K,
            "retention": RETENTION, "g": "N (dense)", "input_dtype": "bf16",
            "l2": "inputs larger than L2 (1.9 GB features, 8.6 GB cost per step)",
            "generator": "paper_2608_13226_gb300.scenes long_video, seeds "
                         f"{rank * B}..{rank * B + B - 1} per rank"}


# --------------------------------------------------------------------------
# reference arm: the oracle timed as it stands
# --------------------------------------------------------------------------
def run_reference(args, rank, world):
    if rank != 0:
        return
    from paper_2608_13226_gb300 import scenes
    s = scenes.make_scene(SCENE_NAME, 0)
    N, D = s["cfg"].N, s["cfg"].D
    K = math.ceil(RETENTION * N - 1e-9)
    import oracle as orc
    orc.build()
    # warm-up steps (untimed) on the scene's first 1024 tokens: they load
    # the library and start its thread pool; every timed step prunes the
    # whole scene
    head = {"feats": s["feats"][:1024], "pos": s["pos"][:1024], "frame": s["frame"][:1024]}
    for _ in range(args.warmup):
        oracle_scene_seconds(head, math.ceil(RETENTION * 1024 - 1e-9))
    times = []
    info = None
    for _ in range(args.steps):
        secs, info = oracle_scene_seconds(s, K)
        times.append(secs)
    scene_s = statistics.mean(times)
    value = 1.0 / scene_s
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "scenes/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(scene_s * 1000.0, 1), "scenes_per_step": 1,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": workload_config(0, SCENES, N, D, K),
            "cpu_baseline": {"value": value, "unit": "scenes/s", "cores": orc.get_threads(),
                             "kind": "oracle",
                             "sample": info["sample"] + "; each timed step is one such "
                                       "scene (scene seed 0); warm-up steps prune its "
                                       "first 1024 tokens",
                             "parts_s": info["parts_s"]},
            "e2e": {"value": value, "unit": "scenes/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# --------------------------------------------------------------------------
# our arm
# --------------------------------------------------------------------------
def run_ours(args, rank, world, local_rank, raw):
    import numpy as np
    import torch

    import paper_2608_13226_gb300 as cp
    from paper_2608_13226_gb300 import build as cuda_build
    cuda_build.build()
    cp.load()
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)

    N, D = 8192, 3584
    K = cp.coverprune_budget(RETENTION, N)
    bits = np.stack([r[0] for r in raw])
    pos_h = np.stack([r[1] for r in raw])
    fr_h = np.stack([r[2] for r in raw])
    B = bits.shape[0]
    feats_pin = torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).pin_memory()
    pos_pin = torch.from_numpy(pos_h).pin_memory()
    fr_pin = torch.from_numpy(fr_h).pin_memory()
    feats = feats_pin.to(dev)
    pos = pos_pin.to(dev)
    fr = fr_pin.to(dev)
    prm = cp.Params()
    stream = torch.cuda.current_stream()

    ws = cp.workspace(cp.CP_OP_SELECT, B, N, D, K, cp.CP_BF16, prm, dev)
    out = {"kept": torch.empty(B, K, dtype=torch.int64, device=dev),
           "objective": torch.empty(B, dtype=torch.float64, device=dev)}

    def step():
        cp.coverprune_select(feats, pos, fr, K, prm, order=False, gains=False, ws=ws, out=out)

    def barrier():
        if dist is not None:
            dist.barrier()
        torch.cuda.synchronize()

    def max_over_ranks(x):
        return reduce_max(x, dist, dev)

    with ClockSampler(local_rank) as clk:
        clk.wait_first_sample()
        for _ in range(args.warmup):
            step()
        barrier()
        cp.coverprune_profile_read()  # clear
        cp.coverprune_profile_enable(True)
        ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        barrier()
        clk.mark(True)
        ev0.record(stream)
        for _ in range(args.steps):
            step()
        ev1.record(stream)
        barrier()
        clk.mark(False)
    cp.coverprune_profile_enable(False)
    prof = cp.coverprune_profile_read()
    clocks = clk.summary()
    st = cp.coverprune_check(ws)
    if st != cp.CP_OK:
        raise RuntimeError(f"device status after the timed region: {cp.status_string(st)}")
    ms_step = max_over_ranks(ev0.elapsed_time(ev1) / args.steps)
    value = whole_job_rate(B, world, ms_step)

    # roofline of the SGS kernel from its own events and its counted reads:
    # the cost bytes its gain evaluations and coverage updates read (the
    # kernel counts them; row blocks known to hold only zero terms are
    # skipped)
    hbm, tf_burst, tf_sust, peak_kind = measured_peaks()
    cstats = cp.coverprune_call_stats(ws)
    sgs_ms, sgs_launches = prof["sgs"]
    launches_per_step = max(sgs_launches // args.steps, 1)
    ldc = (N + 3) // 4 * 4
    sgs_bytes_per_step = cstats["cost_bytes_read"]
    sgs_launch_ms = sgs_ms / max(sgs_launches, 1)
    sgs_gbs = (sgs_bytes_per_step / launches_per_step) / (sgs_launch_ms / 1000.0) / 1e9
    roofline_sgs = {"bound": "hbm", "kernel": "k_sgs_lazy_cl", "achieved": round(sgs_gbs, 1),
                    "peak": hbm, "unit": "GB/s", "frac": round(sgs_gbs / hbm, 4),
                    "frac_of_nominal": round(sgs_gbs / HBM_NOMINAL_GBS, 4),
                    "traffic": read_traffic("k_sgs_lazy", sgs_bytes_per_step // launches_per_step),
                    "peak_source": peak_kind,
                    "algorithmic_bytes_per_launch": sgs_bytes_per_step // launches_per_step,
                    "avg_launch_ms": round(sgs_launch_ms, 3),
                    "gain_evaluations_per_step": cstats["gain_evaluations"],
                    "rounds_per_step": cstats["rounds"],
                    "cost_bytes_read_per_step": cstats["cost_bytes_read"],
                    "full_sweep_evaluations_per_step": B * (K * N - K * (K - 1) // 2)}
    def per_launch_ms(stage):
        ms, launches = prof[stage]
        return ms / launches if ms > 0 and launches > 0 else None

    # the normaliser Gram (tensor cores): the pairs i <= j once, and it also
    # stores their cosines (the upper triangle of [B][N][ldc] fp32) for the
    # cost pass
    gram_ms = per_launch_ms("gram")
    gram_launches_per_step = max(prof["gram"][1] // args.steps, 1)
    gram_flops = B * N * (N + 1) * D // gram_launches_per_step
    gram_tf = gram_flops / (gram_ms / 1000.0) / 1e12 if gram_ms else None
    # the cost pass (HBM): reads the cosines and writes the cost in place
    cost_ms = per_launch_ms("cost")
    cost_launches_per_step = max(prof["cost"][1] // args.steps, 1)
    # the upper triangle of cosines read once, every cost written once, and
    # each token's position, frame and capacity once
    upper = B * (N * (N + 1) // 2 + N * (ldc - N)) * 4
    cost_bytes = (upper + B * N * ldc * 4 + B * N * (16 + 4 + 4)) // cost_launches_per_step
    cost_gbs = cost_bytes / (cost_ms / 1000.0) / 1e9 if cost_ms else None
    roofline_front = {
        "normaliser_gemm": {"bound": "tensor", "kernel": "k_gram_tc", "unit": "TFLOP/s",
                            "achieved": gram_tf and round(gram_tf, 1), "peak": tf_burst,
                            "frac": gram_tf and round(gram_tf / tf_burst, 4),
                            "flops_per_launch": gram_flops,
                            "cosine_bytes_stored_per_launch": upper // gram_launches_per_step,
                            "avg_launch_ms": gram_ms and round(gram_ms, 3)},
        "fst_cost": {"bound": "hbm", "kernel": "k_fst_pair", "unit": "GB/s",
                     "achieved": cost_gbs and round(cost_gbs, 1), "peak": hbm,
                     "frac": cost_gbs and round(cost_gbs / hbm, 4),
                     "frac_of_nominal": cost_gbs and round(cost_gbs / HBM_NOMINAL_GBS, 4),
                     "algorithmic_bytes_per_launch": cost_bytes,
                     "traffic": read_traffic("k_fst_pair", cost_bytes),
                     "avg_launch_ms": cost_ms and round(cost_ms, 3)},
        "peak_source": peak_kind}
    # the line's roofline is the kernel with the largest share of the step
    shares = {"sgs": prof["sgs"][0], "gram": prof["gram"][0], "cost": prof["cost"][0]}
    top = max(shares, key=shares.get)
    if top == "sgs":
        roofline = roofline_sgs
    elif top == "gram":
        r = roofline_front["normaliser_gemm"]
        roofline = {"bound": "tensor", "kernel": r["kernel"], "achieved": r["achieved"],
                    "peak": tf_burst, "unit": "TFLOP/s", "frac": r["frac"], "traffic": None,
                    "peak_source": peak_kind, "algorithmic_flops_per_launch": gram_flops}
    else:
        r = roofline_front["fst_cost"]
        roofline = {"bound": "hbm", "kernel": r["kernel"], "achieved": r["achieved"],
                    "peak": hbm, "unit": "GB/s", "frac": r["frac"], "traffic": r["traffic"],
                    "peak_source": peak_kind, "algorithmic_bytes_per_launch": cost_bytes}

    # end to end through the C ABI with host buffers, as a serving loop runs
    # it: every step uploads its inputs from pinned host memory (on a copy
    # stream, into one of two device input sets, while the previous step
    # computes), calls coverprune_select and reads the kept indices and
    # objectives back.  The timed region spans the first upload to the last
    # read-back.
    kept_pin = torch.empty(B, K, dtype=torch.int64).pin_memory()
    obj_pin = torch.empty(B, dtype=torch.float64).pin_memory()
    inputs = [(torch.empty_like(feats), torch.empty_like(pos), torch.empty_like(fr))
              for _ in range(2)]
    copy_stream = torch.cuda.Stream()
    n_e2e = max(16, args.steps)  # the first upload (not overlapped) amortised over 16 steps
    loaded = [torch.cuda.Event() for _ in range(2)]   # inputs of a set uploaded
    consumed = [torch.cuda.Event() for _ in range(2)]  # a set's step has run

    def upload(i):
        f_dev, p_dev, t_dev = inputs[i % 2]
        with torch.cuda.stream(copy_stream):
            if i >= 2:
                copy_stream.wait_event(consumed[i % 2])
            for sc in range(B):  # one copy a scene, as scenes arrive
                f_dev[sc].copy_(feats_pin[sc], non_blocking=True)
            p_dev.copy_(pos_pin, non_blocking=True)
            t_dev.copy_(fr_pin, non_blocking=True)
            loaded[i % 2].record(copy_stream)

    def run(i):
        f_dev, p_dev, t_dev = inputs[i % 2]
        stream.wait_event(loaded[i % 2])
        cp.coverprune_select(f_dev, p_dev, t_dev, K, prm, order=False, gains=False, ws=ws,
                             out=out)
        consumed[i % 2].record(stream)
        kept_pin.copy_(out["kept"], non_blocking=True)
        obj_pin.copy_(out["objective"], non_blocking=True)

    upload(0)  # warm
    run(0)
    torch.cuda.synchronize()
    barrier()
    a = torch.cuda.Event(enable_timing=True)
    b_ = torch.cuda.Event(enable_timing=True)
    a.record(copy_stream)
    upload(0)
    for i in range(n_e2e):
        if i + 1 < n_e2e:
            upload(i + 1)
        run(i)
    b_.record(stream)
    torch.cuda.synchronize()
    barrier()
    e2e_ms = max_over_ranks(a.elapsed_time(b_) / n_e2e)
    h2d = feats_pin.numel() * 2 + pos_pin.numel() * 4 + fr_pin.numel() * 4
    d2h = kept_pin.numel() * 8 + obj_pin.numel() * 8
    # the upload alone, for context (host-to-device bandwidth of this machine;
    # the best of three copies)
    h2d_gbs = 0.0
    for _ in range(3):
        c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        c0.record(stream)
        inputs[0][0].copy_(feats_pin, non_blocking=True)
        c1.record(stream)
        torch.cuda.synchronize()
        h2d_gbs = max(h2d_gbs, feats_pin.numel() * 2 / (c0.elapsed_time(c1) / 1000.0) / 1e9)
    e2e = {"value": B * world / (e2e_ms / 1000.0), "unit": "scenes/s",
           "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": round(e2e_ms, 3),
           "steps": n_e2e, "h2d_GBps": round(h2d_gbs, 1),
           "overlap": "next step's upload (one copy a scene) on a copy stream during this "
                      "step's selection"}
    del inputs

    # the full sweep (every gain every step), same picks: its HBM roofline
    prm_full = cp.Params(sgs_mode=1)
    cp.coverprune_select(feats, pos, fr, K, prm_full, order=False, gains=False, ws=ws, out=out)
    barrier()
    cp.coverprune_profile_read()
    cp.coverprune_profile_enable(True)
    full_steps = 2
    for _ in range(full_steps):
        cp.coverprune_select(feats, pos, fr, K, prm_full, order=False, gains=False, ws=ws, out=out)
    barrier()
    cp.coverprune_profile_enable(False)
    fprof = cp.coverprune_profile_read()
    fstats = cp.coverprune_call_stats(ws)
    f_ms = fprof["sgs"][0] / max(fprof["sgs"][1], 1)
    f_bytes = fstats["cost_bytes_read"]
    f_gbs = f_bytes / (f_ms / 1000.0) / 1e9
    sweep = {"bound": "hbm", "kernel": "k_sgs<0>", "achieved": round(f_gbs, 1), "peak": hbm,
             "unit": "GB/s", "frac": round(f_gbs / hbm, 4),
             "frac_of_nominal": round(f_gbs / HBM_NOMINAL_GBS, 4),
             "traffic": read_traffic("k_sgs", f_bytes),
             "algorithmic_bytes_per_launch": f_bytes, "avg_launch_ms": round(f_ms, 3)}
    stages = {k: round(v[0] / args.steps, 3) for k, v in prof.items() if v[0] > 0}
    gpu_launches = sum(v[1] for v in prof.values())

    # every other workload: single-scene latencies of the tiny, short-clip,
    # long-video and Lite scenes, and the 32-scene batch at every retention
    # of the sweep (SGS and Lite)
    configs = measure_configs(args, dev, stream, barrier, max_over_ranks, feats, pos, fr, world,
                              {K: {"ms_per_step": ms_step, "stages_ms": {
                                  k: round(v[0] / args.steps, 3) for k, v in prof.items()
                                  if v[0] > 0}, "cost_bytes_read": cstats["cost_bytes_read"]}},
                              hbm)
    latency_ms = configs["long_video"]["select"]["latency_ms"]
    local = configs["batch32_sweep"]["15%"]["select_local_g64"]


    if rank != 0:
        if dist is not None:
            dist.barrier()
            dist.destroy_process_group()
        return
    cpu = None
    if world == 1:
        s0 = {"feats": (bits[0].astype(np.uint32) << 16).view(np.float32), "pos": pos_h[0],
              "frame": fr_h[0]}
        cpu = cpu_baseline_line(s0, K)
    line = {"metric": METRIC, "value": value, "unit": "scenes/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_step, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic",
            "config": workload_config(rank, B, N, D, K),
            "latency_ms": round(latency_ms, 3), "scenes_per_step": B,
            "local_sgs": local, "configs": configs, "roofline": roofline,
            "roofline_sgs": roofline_sgs,
            "roofline_front": roofline_front, "sgs_full_sweep": sweep,
            "stages_ms": stages, "gpu_launches": gpu_launches, "e2e": e2e,
            "clocks": clocks, "cpu_baseline": cpu}
    print(json.dumps(line), flush=True)
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()


# --------------------------------------------------------------------------
# every workload: single-scene latency and the retention sweep
# --------------------------------------------------------------------------
def _event_pair():
    import torch
    return torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)


def timed_calls(call, steps, warmup, stream, sync):
    """(ms per call, per-stage ms per call, launches per call) of `call`
    repeated back to back, CUDA events on the launching stream."""
    import paper_2608_13226_gb300 as cp
    for _ in range(warmup):
        call()
    sync()
    cp.coverprune_profile_read()
    cp.coverprune_profile_enable(True)
    a, b = _event_pair()
    a.record(stream)
    for _ in range(steps):
        call()
    b.record(stream)
    sync()
    cp.coverprune_profile_enable(False)
    prof = cp.coverprune_profile_read()
    return (a.elapsed_time(b) / steps,
            {k: round(v[0] / steps, 3) for k, v in prof.items() if v[0] > 0},
            sum(v[1] for v in prof.values()) / steps)


def latency_of(call, stream, reps=5, warmup=2):
    """Median latency of one call (each timed alone, synchronised on both
    sides) and its per-stage split."""
    import torch

    import paper_2608_13226_gb300 as cp
    for _ in range(warmup):
        call()
    torch.cuda.synchronize()
    cp.coverprune_profile_read()
    cp.coverprune_profile_enable(True)
    lat = []
    for _ in range(reps):
        a, b = _event_pair()
        a.record(stream)
        call()
        b.record(stream)
        torch.cuda.synchronize()
        lat.append(a.elapsed_time(b))
    cp.coverprune_profile_enable(False)
    prof = cp.coverprune_profile_read()
    return statistics.median(lat), {k: round(v[0] / reps, 3) for k, v in prof.items() if v[0] > 0}


def sgs_numbers(stages, K, cost_bytes, hbm):
    """Per-greedy-step time of the selection kernel and the HBM rate of the
    cost bytes it read (its counted reads: gain evaluations and updates)."""
    sgs_ms = stages.get("sgs")
    if not sgs_ms:
        return {}
    out = {"sgs_ms": sgs_ms, "us_per_greedy_step": round(1000.0 * sgs_ms / K, 3)}
    if cost_bytes:
        gbs = cost_bytes / (sgs_ms / 1000.0) / 1e9
        out.update({"sgs_cost_bytes_read": cost_bytes, "sgs_GBps": round(gbs, 1),
                    "sgs_hbm_frac": round(gbs / hbm, 4)})
    return out


def measure_configs(args, dev, stream, sync, max_over_ranks, feats, pos, fr, world, known, hbm):
    """Every workload besides the headline step:

    - single-scene latency (SGS dense; the long video also with g = 64; Lite
      with the min-max and with the bounded feature normaliser) of the tiny
      (N=1024, D=256 fp32, K=102), short-clip (N=4096, D=1280, K=410),
      long-video (N=8192, D=3584, K=1229) and Lite (N=16384, D=3584,
      K=1638) scenes, with the stage split; tiny and short clip hold their
      whole cost matrix in L2 (4 and 67 MB against 129 MB);
    - the 32-scene batch at 5/10/15/25% retention (K = 410/820/1229/2048):
      dense SGS, local SGS (g = 64, 15% only) and Lite both ways, scenes/s
      with the stage split, the selection's time per greedy step and HBM
      rate, and each path's floor (dense SGS: the full sweep's N^2 4 B per
      scene-step at the measured copy bandwidth; Lite: one read of the
      features)."""
    import dataclasses as dc

    import torch

    import paper_2608_13226_gb300 as cp
    from paper_2608_13226_gb300 import scenes
    out = {}
    prm = cp.Params()
    bounded = dc.replace(prm, norm_mode=1)

    def select_call(f, p_, t_, K, prm_s):
        B = f.shape[0] if f.dim() == 3 else 1
        N, D = f.shape[-2], f.shape[-1]
        dt = cp.CP_BF16 if f.dtype == torch.bfloat16 else cp.CP_F32
        ws = cp.workspace(cp.CP_OP_SELECT, B, N, D, K, dt, prm_s, dev)
        o = {"kept": torch.empty(*([B] if f.dim() == 3 else []), K, dtype=torch.int64,
                                 device=dev)}

        def call():
            cp.coverprune_select(f, p_, t_, K, prm_s, order=False, gains=False, objective=False,
                                 ws=ws, out=o)
        return call, ws

    def lite_call(f, p_, t_, K, prm_l):
        B = f.shape[0] if f.dim() == 3 else 1
        N, D = f.shape[-2], f.shape[-1]
        dt = cp.CP_BF16 if f.dtype == torch.bfloat16 else cp.CP_F32
        ws = cp.workspace(cp.CP_OP_LITE, B, N, D, K, dt, prm_l, dev)
        o = {"kept": torch.empty(*([B] if f.dim() == 3 else []), K, dtype=torch.int64,
                                 device=dev)}

        def call():
            cp.coverprune_lite_select(f, p_, t_, K, prm_l, group_start=False, objective=False,
                                      ws=ws, out=o)
        return call, ws

    def check(ws, what):
        st = cp.coverprune_check(ws)
        if st != cp.CP_OK:
            raise RuntimeError(f"device status after {what}: {cp.status_string(st)}")

    def two_in_flight(K, prm_s, n):
        """ms per call with two batches in flight: calls alternate between two
        streams, each with its own workspace, so one call's greedy selection
        (which leaves SMs idle: a block a scene for local SGS, 128 of 152 SMs
        for the dense one) overlaps the next call's front end.  CUDA events:
        from a start both streams wait on to the later of their two ends."""
        streams = [torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)]
        calls = [select_call(feats, pos, fr, K, prm_s) for _ in range(2)]

        def run(i):
            with torch.cuda.stream(streams[i % 2]):
                calls[i % 2][0]()
        for i in range(4):  # warm-up
            run(i)
        sync()
        t0 = torch.cuda.Event(enable_timing=True)
        ends = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
        t0.record(streams[0])
        streams[1].wait_event(t0)
        for i in range(n):
            run(i)
        for k in range(2):
            ends[k].record(streams[k])
        sync()
        ms = max(t0.elapsed_time(e) for e in ends) / n
        for _, w in calls:
            check(w, "two calls in flight")
        return ms

    # ---- single scenes
    for name in ("tiny", "short_clip", "long_video", "lite_long"):
        if name == "long_video":
            f, p_, t_ = feats[0], pos[0], fr[0]
            cfg = scenes.CONFIGS[name]
        else:
            sc = scenes.make_scene(name, 0)
            cfg = sc["cfg"]
            ft = torch.from_numpy(sc["feats"])
            f = (ft.to(torch.bfloat16) if cfg.dtype == "bf16" else ft).to(dev).contiguous()
            p_ = torch.from_numpy(sc["pos"]).to(dev).contiguous()
            t_ = torch.from_numpy(sc["frame"]).to(dev).contiguous()
        N, D, K = cfg.N, cfg.D, cfg.K
        ldc = (N + 3) // 4 * 4
        ent = {"N": N, "D": D, "K": K, "input_dtype": cfg.dtype,
               "l2_resident": N * ldc * 4 + N * D * (2 if cfg.dtype == "bf16" else 4) < 129e6}
        runs = [("select", select_call, prm)] if name != "lite_long" else []
        if name == "long_video":
            runs.append(("select_local_g64", select_call, cp.Params(g=LOCAL_G)))
        if name != "lite_long":  # the rule as Sec. 3.5 prints it (entropic OT residual)
            runs.append(("select_literal", select_call, cp.Params(sgs_mode=2)))
        runs += [("lite", lite_call, prm), ("lite_bounded", lite_call, bounded)]
        for key, mk, pr in runs:
            call, ws = mk(f, p_, t_, K, pr)
            slow = key == "select_literal" and N > 4096
            ms, stages = latency_of(call, stream, reps=2 if slow else 5, warmup=1 if slow else 2)
            check(ws, f"{name} {key}")
            r = {"latency_ms": round(ms, 3), "stages_ms": stages}
            if key.startswith("select"):
                r.update(sgs_numbers(stages, K, None, hbm))
            if key == "select_literal":
                r.update({"sot_eps": pr.sot_eps, "sot_iters": pr.sot_iters,
                          "rule": "Eqs. greedy_flow / sgs_select as printed (sgs_mode 2)"})
            out.setdefault(name, ent)[key] = r
            del ws
        del f, p_, t_

    # ---- the 32-scene batch at every retention
    B, N, D = feats.shape
    sweep = {}
    for R in scenes.BATCH32_RETENTION:
        K = cp.coverprune_budget(R, N)
        e = {"K": K}
        if K in known:
            ms, stages, cbytes = (known[K]["ms_per_step"], known[K]["stages_ms"],
                                  known[K]["cost_bytes_read"])
        else:
            call, ws = select_call(feats, pos, fr, K, prm)
            ms, stages, _ = timed_calls(call, args.steps, args.warmup, stream, sync)
            check(ws, f"batch select K={K}")
            cbytes = cp.coverprune_call_stats(ws)["cost_bytes_read"]
            del ws
        ms = max_over_ranks(ms)
        full_sweep_ms = B * K * N * N * 4 / (hbm * 1e9) * 1e3
        e["select"] = dict({"scenes_per_s": B * world / (ms / 1000.0), "ms_per_step": round(ms, 3),
                            "stages_ms": stages,
                            "full_sweep_floor_ms": round(full_sweep_ms, 1)},
                           **sgs_numbers(stages, K, cbytes, hbm))
        if abs(R - RETENTION) < 1e-9:
            # local SGS: with the min-max normaliser (the all-pairs Gram runs
            # for the feature range and stores every cosine), and with the
            # bounded one (only the Morton tiles holding a neighbour pair)
            for key, pl in (("select_local_g64", cp.Params(g=LOCAL_G)),
                            ("select_local_g64_bounded", cp.Params(g=LOCAL_G, norm_mode=1))):
                call, ws = select_call(feats, pos, fr, K, pl)
                ms, stages, _ = timed_calls(call, args.steps, args.warmup, stream, sync)
                check(ws, f"batch {key}")
                gst = cp.coverprune_call_stats(ws)
                ms = max_over_ranks(ms)
                e[key] = dict({"g": LOCAL_G, "scenes_per_s": B * world / (ms / 1000.0),
                               "ms_per_step": round(ms, 3), "stages_ms": stages,
                               "gain_evaluations_per_step": gst["gain_evaluations"]},
                              **sgs_numbers(stages, K, None, hbm))
                del ws
            two = {}
            for key, pl in (("select", prm), ("select_local_g64", cp.Params(g=LOCAL_G)),
                            ("select_local_g64_bounded", cp.Params(g=LOCAL_G, norm_mode=1))):
                ms = max_over_ranks(two_in_flight(K, pl, max(8, args.steps)))
                two[key] = {"scenes_per_s": B * world / (ms / 1000.0), "ms_per_step": round(ms, 3)}
            e["two_batches_in_flight"] = two
        floor_ms = B * N * D * 2 / (hbm * 1e9) * 1e3  # one read of the features
        for key, pr in (("lite", prm), ("lite_bounded", bounded)):
            call, ws = lite_call(feats, pos, fr, K, pr)
            ms, stages, _ = timed_calls(call, args.steps, args.warmup, stream, sync)
            check(ws, f"batch {key} K={K}")
            ms = max_over_ranks(ms)
            e[key] = {"scenes_per_s": B * world / (ms / 1000.0), "ms_per_step": round(ms, 3),
                      "stages_ms": stages, "feature_read_floor_ms": round(floor_ms, 3),
                      "frac_of_floor": round(floor_ms / ms, 4)}
            del ws
        sweep[f"{round(R * 100)}%"] = e
    out["batch32_sweep"] = sweep
    out["notes"] = ("bounded = the bounded feature normaliser (d_f / 2), no all-pairs Gram; "
                    "latency = one call timed alone (median of 5 after 2 warm-ups); "
                    "batch numbers: CUDA events over back-to-back calls on resident inputs; "
                    "two_batches_in_flight: the same calls alternating between two streams "
                    "with a workspace each (a serving loop with two batches in flight)")
    return out


def read_traffic(kernel: str, algorithmic_bytes: int):
    """DRAM bytes of one launch of `kernel`, scaled from the committed ncu
    record of that kernel (profiles/<kernel>_traffic.txt: its DRAM bytes per
    algorithmic byte on a captured launch, and the sources it was built
    from) by this launch's algorithmic bytes; None when no record exists or
    those sources have changed since the counters were taken."""
    import hashlib
    path = os.path.join(ROOT, "profiles", f"{kernel}_traffic.txt")
    try:
        rec = {}
        for line in open(path):
            if ":" in line and not line.startswith("#"):
                k, v = line.split(":", 1)
                rec[k.strip()] = v.strip()
        files = rec.get("source_files", "sgs.cu common.cuh").split()
        src = b"".join(open(os.path.join(ROOT, "paper_2608_13226_gb300", "csrc", f), "rb").read()
                       for f in files)
        if hashlib.sha256(src).hexdigest()[:16] != rec.get("source_sha256"):
            return None
        return round(float(rec["dram_bytes_per_algorithmic_byte"]) * algorithmic_bytes)
    except (OSError, KeyError, ValueError):
        return None


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    args = ap.parse_args()
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    # scenes are drawn in a spawned pool before any CUDA use
    raw = make_batch(rank_seeds(rank))
    run_ours(args, rank, world, local_rank, raw)


if __name__ == "__main__":
    main()
