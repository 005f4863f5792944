"""Seeded synthetic 3D scenes shaped like the paper's workloads.

The paper evaluates on multi-view indoor video (32 uniformly sampled frames,
Sec. 5.1) whose visual tokens carry a feature, a 3D coordinate and a frame
index (Sec. 3.2).  No dataset or trained encoder is available, so these scenes
stand in for them: repeated observations of the same surfaces share a feature
mode, cluster sizes are heavy-tailed and 5% of tokens are outliers.

This module serves both the CUDA path's tests/benchmark and the CPU oracle.
It holds none of the method's arithmetic (no cost, capacity, neighbour search,
Morton order or selection); it only draws numbers.

Named workloads (token counts, feature widths and budgets):
  tiny        N=1024 (8 frames x 128), D=256 fp32, 16-mode mixture,
              per-mode position blobs in an 8x8x3 m box, K=102
  short_clip  N=4096 (16 x 256), D=1280 bf16, 32 equal modes, depth
              back-projection along a circular camera path, K=410
  long_video  N=8192 (32 x 256), D=3584 bf16, 64 modes with Zipf(1.2) sizes,
              random-walk camera, K=1229 (15%)
  lite_long   N=16384 (64 x 256), D=3584 bf16, long_video generator, K=1638
  batch32     32 long_video scenes (seeds 0..31); retention 5/10/15/25%
"""
from __future__ import annotations

import math
from dataclasses import dataclass, replace

import numpy as np

ROOM = (8.0, 8.0, 3.0)


@dataclass(frozen=True)
class SceneConfig:
    name: str
    N: int
    tokens_per_frame: int
    D: int
    dtype: str          # "f32" or "bf16"
    modes: int
    zipf: float | None  # None = equal-probability modes
    positions: str      # "blobs" | "circle" | "walk"
    K: int
    outlier_frac: float = 0.05
    sigma_f: float = 0.3
    sigma_x: float = 0.3


CONFIGS = {
    "tiny": SceneConfig("tiny", 1024, 128, 256, "f32", 16, None, "blobs", 102),
    "short_clip": SceneConfig("short_clip", 4096, 256, 1280, "bf16", 32, None, "circle", 410),
    "long_video": SceneConfig("long_video", 8192, 256, 3584, "bf16", 64, 1.2, "walk", 1229),
    "lite_long": SceneConfig("lite_long", 16384, 256, 3584, "bf16", 64, 1.2, "walk", 1638),
}
BATCH32_RETENTION = (0.05, 0.10, 0.15, 0.25)


def config(name: str, **override) -> SceneConfig:
    cfg = CONFIGS[name]
    return replace(cfg, **override) if override else cfg


def round_to_bf16(a: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bfloat16 (ties to even); returns
    float32 holding bf16-representable values."""
    u = np.array(a, dtype=np.float32, copy=True).view(np.uint32)
    bias = u >> 16
    bias &= np.uint32(1)
    bias += np.uint32(0x7FFF)
    u += bias
    u &= np.uint32(0xFFFF0000)
    return u.view(np.float32)


def bf16_bits(a: np.ndarray) -> np.ndarray:
    """uint16 bit patterns of bf16-representable float32 values."""
    return (np.ascontiguousarray(a, dtype=np.float32).view(np.uint32) >> 16).astype(np.uint16)


def _mode_sizes(rng, cfg: SceneConfig, n: int) -> np.ndarray:
    if cfg.zipf is None:
        w = np.ones(cfg.modes)
    else:
        w = np.arange(1, cfg.modes + 1, dtype=np.float64) ** (-cfg.zipf)
    share = w / w.sum() * n
    sizes = np.floor(share).astype(np.int64)
    rest = n - sizes.sum()
    if rest > 0:  # largest remainder
        sizes[np.argsort(-(share - sizes), kind="stable")[:rest]] += 1
    return sizes


def _camera_path(rng, cfg: SceneConfig, frames: int):
    cx, cy = ROOM[0] / 2, ROOM[1] / 2
    if cfg.positions == "circle":
        ang = 2 * math.pi * np.arange(frames) / frames
        xy = np.stack([cx + 2.0 * np.cos(ang), cy + 2.0 * np.sin(ang)], axis=1)
        yaw = ang + math.pi / 2
    else:  # random walk
        xy = np.empty((frames, 2))
        yaw = np.empty(frames)
        xy[0] = (cx, cy)
        yaw[0] = rng.uniform(0, 2 * math.pi)
        for f in range(1, frames):
            xy[f] = np.clip(xy[f - 1] + rng.normal(0, 0.25, 2), 1.0, 7.0)
            yaw[f] = yaw[f - 1] + rng.normal(0, math.radians(20))
    return xy, yaw


def _backprojected_points(rng, cfg: SceneConfig) -> np.ndarray:
    """One token per image patch (square patch grid per frame), pinhole with
    a 90 degree field of view, depth = distance to the room's walls clipped
    to [1, 6] m with 2% multiplicative noise."""
    tpf = cfg.tokens_per_frame
    side = int(round(math.sqrt(tpf)))
    assert side * side == tpf, "tokens_per_frame must be a square"
    frames = -(-cfg.N // tpf)
    xy, yaw = _camera_path(rng, cfg, frames)
    u = (np.arange(side) + 0.5) / side * 2 - 1
    uu, vv = np.meshgrid(u, u, indexing="xy")
    uu, vv = uu.ravel(), vv.ravel()
    pts = np.empty((frames * tpf, 3))
    room = np.array(ROOM)
    for f in range(frames):
        c, s = math.cos(yaw[f]), math.sin(yaw[f])
        fwd = np.array([c, s, 0.0])
        right = np.array([s, -c, 0.0])
        up = np.array([0.0, 0.0, 1.0])
        d = fwd[None] + uu[:, None] * right[None] - vv[:, None] * up[None]
        d /= np.linalg.norm(d, axis=1, keepdims=True)
        p = np.array([xy[f, 0], xy[f, 1], 1.5])
        with np.errstate(divide="ignore"):
            t_hi = np.where(d > 0, (room[None] - p[None]) / d, np.inf)
            t_lo = np.where(d < 0, (0.0 - p[None]) / d, np.inf)
        t = np.minimum(t_hi, t_lo).min(axis=1)
        depth = np.clip(t, 1.0, 6.0) * (1.0 + rng.normal(0, 0.02, tpf))
        pts[f * tpf:(f + 1) * tpf] = p[None] + depth[:, None] * d
    return pts[:cfg.N]


def make_scene(cfg: SceneConfig | str, seed: int = 0) -> dict:
    """One scene: feats float32 [N, D] (bf16-rounded when cfg.dtype == "bf16"),
    pos float32 [N, 3] metres, frame int32 [N] (token // tokens_per_frame)."""
    if isinstance(cfg, str):
        cfg = CONFIGS[cfg]
    rng = np.random.default_rng(seed)
    N, D = cfg.N, cfg.D
    n_out = int(round(cfg.outlier_frac * N))
    outliers = np.zeros(N, dtype=bool)
    outliers[rng.choice(N, n_out, replace=False)] = True
    inliers = np.flatnonzero(~outliers)

    centres = rng.standard_normal((cfg.modes, D), dtype=np.float32)
    centres /= np.linalg.norm(centres, axis=1, keepdims=True)

    label = np.full(N, -1, dtype=np.int64)
    if cfg.positions == "blobs":
        blob = rng.uniform(0, 1, (cfg.modes, 3)) * np.array(ROOM)
        label[inliers] = rng.integers(cfg.modes, size=inliers.size)
        pos = blob[np.maximum(label, 0)] + rng.normal(0, cfg.sigma_x, (N, 3))
        pos[outliers] = rng.uniform(0, 1, (n_out, 3)) * np.array(ROOM)
        pos = np.clip(pos, 0, np.array(ROOM))
    else:
        pos = _backprojected_points(rng, cfg)
        # surfaces seen from several frames share a feature mode: order the
        # inliers by (height band, azimuth about the room centre) and give
        # contiguous runs the modes in a shuffled order
        rel = pos[inliers] - np.array([ROOM[0] / 2, ROOM[1] / 2, 0.0])
        band = np.clip(np.floor(pos[inliers, 2]), 0, 2)
        key = band * 10.0 + (np.arctan2(rel[:, 1], rel[:, 0]) + math.pi)
        ordered = inliers[np.argsort(key, kind="stable")]
        sizes = _mode_sizes(rng, cfg, inliers.size)
        modes = rng.permutation(cfg.modes)
        label[ordered] = np.repeat(modes, sizes)

    feats = rng.standard_normal((N, D), dtype=np.float32)
    feats *= np.float32(cfg.sigma_f / math.sqrt(D))
    feats += centres[np.maximum(label, 0)]
    out_f = rng.random((n_out, D), dtype=np.float32)
    out_f *= np.float32(2.0 * math.sqrt(3.0 / D))
    out_f -= np.float32(math.sqrt(3.0 / D))
    feats[outliers] = out_f
    if cfg.dtype == "bf16":
        feats = round_to_bf16(feats)
    frame = (np.arange(N) // cfg.tokens_per_frame).astype(np.int32)
    return {"name": cfg.name, "cfg": cfg, "seed": seed, "feats": feats,
            "pos": pos.astype(np.float32), "frame": frame, "label": label,
            "dtype": cfg.dtype, "K": cfg.K}


def make_batch(cfg: SceneConfig | str, seeds) -> dict:
    """Independent scenes stacked: feats [B, N, D], pos [B, N, 3], frame [B, N]."""
    scenes = [make_scene(cfg, s) for s in seeds]
    return {"feats": np.stack([s["feats"] for s in scenes]),
            "pos": np.stack([s["pos"] for s in scenes]),
            "frame": np.stack([s["frame"] for s in scenes]),
            "dtype": scenes[0]["dtype"], "cfg": scenes[0]["cfg"], "seeds": list(seeds)}
