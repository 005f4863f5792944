"""The seeded scene generator: deterministic, shaped like the named
workloads, bf16 rounding identical to torch's."""
import numpy as np
import pytest
import torch

from paper_2608_13226_gb300 import scenes


@pytest.mark.parametrize("name", ["tiny", "short_clip"])
def test_deterministic_and_shaped(name):
    a = scenes.make_scene(name, 3)
    b = scenes.make_scene(name, 3)
    c = scenes.make_scene(name, 4)
    cfg = scenes.CONFIGS[name]
    for k in ("feats", "pos", "frame"):
        np.testing.assert_array_equal(a[k], b[k])
    assert not np.array_equal(a["feats"], c["feats"])
    assert a["feats"].shape == (cfg.N, cfg.D) and a["feats"].dtype == np.float32
    assert a["pos"].shape == (cfg.N, 3) and a["pos"].dtype == np.float32
    assert a["frame"].dtype == np.int32
    np.testing.assert_array_equal(a["frame"], np.arange(cfg.N) // cfg.tokens_per_frame)
    assert a["K"] == cfg.K
    n_out = int(round(0.05 * cfg.N))
    assert (a["label"] < 0).sum() == n_out
    assert np.isfinite(a["feats"]).all() and np.isfinite(a["pos"]).all()


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(0)
    x = (rng.standard_normal(100000) * np.exp(rng.uniform(-20, 20, 100000))).astype(np.float32)
    ours = scenes.round_to_bf16(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float32).numpy()
    np.testing.assert_array_equal(ours, ref)
    bits = scenes.bf16_bits(ours)
    back = torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).float().numpy()
    np.testing.assert_array_equal(back, ours)


def test_short_clip_positions_and_modes():
    s = scenes.make_scene("short_clip", 0)
    p = s["pos"]
    # back-projected points sit near the 8 x 8 x 3 m room's walls
    assert p[:, 0].min() > -1 and p[:, 0].max() < 9
    assert p[:, 2].min() > -1 and p[:, 2].max() < 4
    lab = s["label"][s["label"] >= 0]
    sizes = np.bincount(lab, minlength=32)
    assert sizes.max() - sizes.min() <= 1  # equal modes


def test_tiny_feature_geometry():
    s = scenes.make_scene("tiny", 0)
    f = s["feats"]
    nrm = np.linalg.norm(f, axis=1)
    assert abs(np.median(nrm) - 1.04) < 0.05  # unit centre + noise of norm 0.3
    inl = s["label"] >= 0
    lab = s["label"][inl]
    cos = (f[inl][:200] @ f[inl][:200].T) / np.outer(nrm[inl][:200], nrm[inl][:200])
    same = lab[:200, None] == lab[None, :200]
    assert cos[same & ~np.eye(200, dtype=bool)].mean() > 0.8
    assert abs(cos[~same].mean()) < 0.1


@pytest.mark.slow
def test_long_video_zipf_sizes():
    s = scenes.make_scene("long_video", 0)
    lab = s["label"][s["label"] >= 0]
    sizes = np.sort(np.bincount(lab, minlength=64))[::-1]
    assert sizes.sum() == 8192 - int(round(0.05 * 8192))
    w = np.arange(1, 65) ** -1.2
    np.testing.assert_allclose(sizes / sizes.sum(), w / w.sum(), atol=2e-3)
