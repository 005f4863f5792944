"""Parity of the CUDA path (through the C ABI) with the CPU oracle on the
same seeded inputs.  Sizes span several tiles and a ragged tail; the bars are
in gpu_util (cost 1e-5 / 1e-3 relative for fp32 / bf16 inputs, kept sets
exact up to near-ties of 1e-5, objective 1e-4)."""
import numpy as np
import pytest
import torch

import paper_2608_13226_gb300 as cp
from gpu_util import (assert_capacity_close, assert_cost_close, batch_to_dev,
                      check_lite_end_to_end, check_sgs_end_to_end, check_sgs_teacher_forced,
                      measured_errors, oracle_params, scene, to_dev)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2608_13226_gb300 import build
    build.build()
    cp.load()
    torch.cuda.init()


def host(t):
    return t.detach().cpu().numpy()


def f64(s):
    return s["feats"].astype(np.float64)


# --------------------------------------------------------------------------
# K1: neighbours (bit-exact)
# --------------------------------------------------------------------------

@pytest.mark.parametrize("name,N,k", [("tiny", 1024, 8), ("short_clip", 4096, 63),
                                      ("long_video", 1000, 17), ("tiny", 37, 36),
                                      ("long_video", 3000, 64), ("long_video", 2000, 65),
                                      ("long_video", 8192, 8), ("long_video", 8192, 63)])
def test_knn_bit_exact(orc, name, N, k):
    s = scene(name, 1, N=N, D=64)
    _, pos, _ = to_dev(s)
    nbr, dia = cp.coverprune_knn(pos, k)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(host(nbr), orc.knn_others(s["pos"], k))
    nm = orc.normalisers(np.ones((N, 1)), s["pos"], s["frame"])
    assert abs(float(dia) - nm.x_hi) <= 1e-6 * nm.x_hi


def test_knn_ties_and_duplicates(orc):
    rng = np.random.default_rng(5)
    X = np.repeat((rng.integers(0, 4, (40, 3)) * 0.5).astype(np.float32), 3, axis=0)  # coincident
    pos = torch.from_numpy(X).cuda()
    nbr, _ = cp.coverprune_knn(pos, 11)
    np.testing.assert_array_equal(host(nbr), orc.knn_others(X, 11))


def _max_d2_fp32(X):
    """The largest squared distance over all pairs, every operation rounded
    in fp32 in the kernels' order ((dx dx + dy dy) + dz dz)."""
    X = np.asarray(X, np.float32)
    best = np.float32(0.0)
    for i0 in range(0, len(X), 512):
        d = X[i0:i0 + 512, None, :] - X[None, :, :]
        sq = d * d
        best = max(best, ((sq[..., 0] + sq[..., 1]) + sq[..., 2]).max())
    return best


def _shapes(rng):
    box = rng.random((3000, 3)).astype(np.float32) * np.float32([8, 6, 3])
    th, ph = rng.random(2500) * 2 * np.pi, np.arccos(rng.uniform(-1, 1, 2500))
    shell = np.stack([np.sin(ph) * np.cos(th), np.sin(ph) * np.sin(th), np.cos(ph)], 1)
    line = np.zeros((700, 3), np.float32)
    line[:, 0] = rng.random(700)
    dup = np.repeat(rng.random((60, 3)).astype(np.float32), 5, axis=0)
    return {"box": box, "walls": scene("long_video", 3, N=2048, D=16)["pos"],
            "shell": (2.5 * shell).astype(np.float32), "line": line, "dup": dup,
            "offset": box[:900] + np.float32(1000.0), "one": box[:1], "two": box[:2],
            "same": np.repeat(box[:1], 33, axis=0)}


@pytest.mark.parametrize("k", [8, 0])
def test_diameter_from_grid_is_exact(k):
    # the grid path (k <= 8) prunes cell pairs by a bound: its diameter must
    # be exactly the largest pinned-fp32 d^2 over all pairs, whatever the shape
    rng = np.random.default_rng(21)
    for name, X in _shapes(rng).items():
        pos = torch.from_numpy(np.ascontiguousarray(X, np.float32)).cuda()
        _, dia = cp.coverprune_knn(pos, min(k, len(X) - 1))
        got = float(host(dia))
        want = float(np.sqrt(np.float32(_max_d2_fp32(X)), dtype=np.float32))
        assert got == want, f"{name}: {got} != {want}"


def test_diameter_grid_equals_brute_force_batched():
    rng = np.random.default_rng(22)
    X = (rng.random((3, 1500, 3)) * np.float32([8, 8, 3])).astype(np.float32)
    X[1, :, 2] = 0.0  # a flat scene
    pos = torch.from_numpy(X).cuda()
    _, dia = cp.coverprune_knn(pos, 8)
    nbr = torch.empty(3, 1500, 8, dtype=torch.int32, device="cuda")
    dia_bf = torch.empty(3, dtype=torch.float32, device="cuda")
    cp.coverprune_knn_noalloc(pos, nbr, dia_bf)
    torch.cuda.synchronize()
    assert torch.equal(dia, dia_bf)


# --------------------------------------------------------------------------
# K0-K4: normalisers, cost, capacity
# --------------------------------------------------------------------------

def _cost_case(orc, s, prm=cp.Params()):
    f, pos, fr = to_dev(s)
    out = cp.coverprune_cost(f, pos, fr, prm)
    torch.cuda.synchronize()
    F = f64(s)
    nm = orc.normalisers(F, s["pos"], s["frame"], prm.norm_mode)
    op = oracle_params(orc, prm)
    Co = orc.cost_matrix(F, s["pos"], s["frame"], op.weights, nm)
    _, vo = orc.capacity(F, s["pos"], s["frame"], op.weights, nm, prm.n_cap, mode=prm.capacity_mode)
    return out, nm, Co, vo


def test_cost_tiny_fp32_full(orc):
    s = scene("tiny", 0)
    out, nm, Co, vo = _cost_case(orc, s)
    ng = host(out["norms"])
    want = [nm.f_lo, nm.f_hi, nm.x_lo, nm.x_hi, nm.tau_lo, nm.tau_hi]
    np.testing.assert_allclose(ng, want, rtol=1e-5, atol=1e-6)
    err = assert_cost_close(host(out["cost"]), Co, "f32")
    print(f"tiny fp32 cost max rel err {err:.3g}")
    assert_capacity_close(host(out["capacity"]), vo, "f32")
    assert np.all(np.diag(host(out["cost"])) == 0.0)


@pytest.mark.parametrize("N,D,seed", [(777, 512, 0), (300, 3584, 1), (1100, 1280, 2)])
def test_cost_bf16_ragged(orc, N, D, seed):
    s = scene("long_video", seed, N=N, D=D)
    out, nm, Co, vo = _cost_case(orc, s)
    err = assert_cost_close(host(out["cost"]), Co, "bf16")
    print(f"bf16 N={N} D={D} cost max rel err {err:.3g}")
    assert_capacity_close(host(out["capacity"]), vo, "bf16")


def test_cost_output_offset_by_one_float():
    """An output whose base is 4-byte but not 16-byte aligned (a slice one
    float into a buffer) gets the same cost as an aligned one: the kernel
    falls back from 16-byte stores when the base or the row stride forbids
    them."""
    s = scene("short_clip", 9, N=256, D=128)
    f, pos, fr = to_dev(s)
    ref = cp.coverprune_cost(f, pos, fr, cp.Params(), capacity=False, norms=False)["cost"]
    buf = torch.full((256 * 256 + 1,), -1.0, dtype=torch.float32, device="cuda")
    shifted = buf[1:].view(256, 256)
    assert shifted.data_ptr() % 16 == 4
    cp.coverprune_cost(f, pos, fr, cp.Params(), capacity=False, norms=False,
                       out={"cost": shifted})
    torch.cuda.synchronize()
    assert torch.equal(shifted, ref)
    assert buf[0].item() == -1.0


def test_cost_ablation_weights(orc):
    s = scene("short_clip", 3, N=500, D=256)
    prm = cp.Params(lambda_f=0.5, lambda_x=2.0, lambda_tau=0.0, kappa=3.0, alpha_f=0.2,
                    alpha_x=1.5, alpha_tau=0.7, n_cap=5)
    out, nm, Co, vo = _cost_case(orc, s, prm)
    assert_cost_close(host(out["cost"]), Co, "bf16")
    assert_capacity_close(host(out["capacity"]), vo, "bf16")
    out1, _, _, vo1 = _cost_case(orc, s, cp.Params(capacity_mode=1))
    np.testing.assert_allclose(host(out1["capacity"]), 1.0 / 500, rtol=1e-7)


@pytest.mark.parametrize("name,N,D,dtype", [("tiny", 1024, 256, "f32"),
                                            ("long_video", 777, 512, "bf16")])
def test_cost_bounded_normaliser(orc, name, N, D, dtype):
    """norm_mode 1: the feature term is d_f / 2; the fp32 path runs without
    the Gram, the bf16 path still takes its cosines from it."""
    s = scene(name, 5, N=N, D=D)
    prm = cp.Params(norm_mode=1)
    out, nm, Co, vo = _cost_case(orc, s, prm)
    ng = host(out["norms"])
    assert ng[0] == 0.0 and ng[1] == 2.0
    np.testing.assert_allclose(ng, [nm.f_lo, nm.f_hi, nm.x_lo, nm.x_hi, nm.tau_lo, nm.tau_hi],
                               rtol=1e-5, atol=1e-6)
    assert_cost_close(host(out["cost"]), Co, dtype)
    assert_capacity_close(host(out["capacity"]), vo, dtype)
    # the min-max cost of the same scene differs (its feature range is < 2)
    ref = cp.coverprune_cost(*to_dev(s), cp.Params(), capacity=False, norms=False)["cost"]
    assert not torch.equal(ref, out["cost"])


def test_sgs_bounded_normaliser_teacher_forced(orc):
    s = scene("short_clip", 6, N=999, D=512)
    K = 200
    prm = cp.Params(norm_mode=1)
    sel, cst = _select_case(orc, s, K, prm)
    order = host(sel["order"])
    check_sgs_teacher_forced(orc, host(cst["cost"]).astype(np.float64),
                             host(cst["capacity"]).astype(np.float64), order, host(sel["gains"]),
                             float(host(sel["objective"])), 3.0, 0, None)
    ora = orc.select(f64(s), s["pos"], s["frame"], K, oracle_params(orc, prm))
    check_sgs_end_to_end(orc, ora, order, host(sel["kept"]), 3.0, 0)


def test_cost_degenerate_scenes(orc):
    # identical tokens: every range is empty, C == 0, v uniform
    N = 130
    s = {"feats": np.tile(np.linspace(-1, 1, 64, dtype=np.float32), (N, 1)),
         "pos": np.tile(np.array([[1.0, 2.0, 3.0]], dtype=np.float32), (N, 1)),
         "frame": np.zeros(N, dtype=np.int32), "dtype": "f32"}
    out, nm, Co, vo = _cost_case(orc, s)
    assert np.all(host(out["cost"]) == 0.0)
    np.testing.assert_allclose(host(out["capacity"]), 1.0 / N, rtol=1e-7)
    # a zero feature (cos := 0), a single frame, two tokens
    rng = np.random.default_rng(9)
    s2 = {"feats": rng.standard_normal((70, 32)).astype(np.float32),
          "pos": rng.random((70, 3)).astype(np.float32),
          "frame": np.zeros(70, dtype=np.int32), "dtype": "f32"}
    s2["feats"][13] = 0.0
    out, nm, Co, vo = _cost_case(orc, s2)
    assert_cost_close(host(out["cost"]), Co, "f32")
    assert_capacity_close(host(out["capacity"]), vo, "f32")
    s3 = {k: (v[:2] if isinstance(v, np.ndarray) else v) for k, v in s2.items()}
    out, nm, Co, vo = _cost_case(orc, s3)
    assert_cost_close(host(out["cost"]), Co, "f32")


# --------------------------------------------------------------------------
# K5: SGS
# --------------------------------------------------------------------------

def _select_case(orc, s, K, prm):
    f, pos, fr = to_dev(s)
    sel = cp.coverprune_select(f, pos, fr, K, prm)
    cst = cp.coverprune_cost(f, pos, fr, prm)
    torch.cuda.synchronize()
    return sel, cst


@pytest.mark.parametrize("g", [0, 16])
def test_sgs_tiny_teacher_forced_and_end_to_end(orc, g):
    s = scene("tiny", 0)
    K = s["K"]
    prm = cp.Params(g=g)
    sel, cst = _select_case(orc, s, K, prm)
    order, kept = host(sel["order"]), host(sel["kept"])
    assert np.array_equal(np.sort(order), kept) and len(set(kept.tolist())) == K
    M0 = 3.0
    nbr = None
    if g:
        nbr = orc.knn_others(s["pos"], g - 1)
    div, _ = check_sgs_teacher_forced(orc, host(cst["cost"]).astype(np.float64),
                                      host(cst["capacity"]).astype(np.float64), order,
                                      host(sel["gains"]), float(host(sel["objective"])), M0, g, nbr)
    ora = orc.select(f64(s), s["pos"], s["frame"], K, oracle_params(orc, prm))
    first, jac = check_sgs_end_to_end(orc, ora, order, kept, M0, g)
    print(f"g={g}: teacher-forced near-tie picks {div}; end-to-end equal for {first}/{K} "
          f"steps, Jaccard {jac:.3f}")


@pytest.mark.parametrize("N,K,g,seed", [(1500, 150, 0, 0), (999, 333, 24, 1), (260, 260, 0, 2)])
def test_sgs_bf16_teacher_forced(orc, N, K, g, seed):
    s = scene("short_clip", seed, N=N, D=512)
    prm = cp.Params(g=g, n_cap=6)
    sel, cst = _select_case(orc, s, K, prm)
    order = host(sel["order"])
    nbr = orc.knn_others(s["pos"], g - 1) if g else None
    check_sgs_teacher_forced(orc, host(cst["cost"]).astype(np.float64),
                             host(cst["capacity"]).astype(np.float64), order, host(sel["gains"]),
                             float(host(sel["objective"])), 3.0, g, nbr)
    gains = host(sel["gains"])
    assert np.all(np.diff(gains) <= 0)  # monotone in fp32 as well (exact min updates)
    if K == N:
        assert host(sel["kept"]).tolist() == list(range(N))
        assert float(host(sel["objective"])) == 0.0


def test_short_clip_full_config(orc):
    """The short-clip workload at its own size (N=4096, D=1280 bf16,
    K=410): the whole cost matrix and capacity against the oracle; the
    greedy teacher-forced over every step on the GPU's own cost and end to
    end against the oracle's greedy on its own cost; Lite teacher-forced on
    the GPU's capacity and end to end against the oracle's Lite."""
    s = scene("short_clip", 0)
    K = s["K"]
    assert (s["feats"].shape, K) == ((4096, 1280), 410)
    prm = cp.Params()
    sel, cst = _select_case(orc, s, K, prm)
    F = f64(s)
    op = oracle_params(orc, prm)
    ora = orc.select(F, s["pos"], s["frame"], K, op)
    assert_cost_close(host(cst["cost"]), ora["C"], "bf16")
    assert_capacity_close(host(cst["capacity"]), ora["v"], "bf16")
    order, kept = host(sel["order"]), host(sel["kept"])
    div, _ = check_sgs_teacher_forced(orc, host(cst["cost"]).astype(np.float64),
                                      host(cst["capacity"]).astype(np.float64),
                                      order, host(sel["gains"]),
                                      float(host(sel["objective"])), 3.0)
    eps = measured_errors(host(cst["cost"]), ora["C"], host(cst["capacity"]), ora["v"])
    first, jac = check_sgs_end_to_end(orc, ora, order, kept, 3.0, eps=eps)
    near = _lite_check(orc, s, K, prm, "bf16")
    f, pos, fr = to_dev(s)
    lt = cp.coverprune_lite_select(f, pos, fr, K, prm)
    torch.cuda.synchronize()
    ora_l = orc.lite(F, s["pos"], s["frame"], K, op)
    moved, near_e = check_lite_end_to_end(orc, s, ora_l, host(lt["kept"]),
                                          host(lt["group_start"]), op.weights)
    print(f"short clip: teacher-forced near-tie picks {div}/{K}, end to end equal for "
          f"{first}/{K} steps (Jaccard {jac:.3f}); Lite near-tie prototypes {near}/{K} forced, "
          f"{near_e} end to end, moved group starts {moved}")


# --------------------------------------------------------------------------
# K5 as Sec. 3.5 prints it (sgs_mode 2): entropic semi-relaxed OT residual
# (Eqs. srpot_sinkhorn, greedy_flow, sgs_select).  The paper fixes neither
# eps nor the iteration count; both sides run the same iterations from the
# same start, the GPU in fp32 and the oracle in fp64.  A saturated column's
# residual is a difference of two nearly equal numbers, so the GPU's carries
# an error of a few fp32 roundings of log-sum-exp terms (~1e-5 of v_j), and a
# score's error is bounded by that fraction of w(t) = sum_{j in M_g(t)} v_j
# C(t, j), the score of t against the full capacity.  Scores are compared
# to LIT_RTOL of (score + w): a bar taken from the fp32 log-sum-exp, not from
# the paper (parity unpinned beyond the oracle's own pins).  Where a whole
# neighbourhood is served (the rule's degenerate case) every score is that
# noise, and the pick among them is arbitrary on both sides.
# --------------------------------------------------------------------------
LIT_RTOL = 1e-4


def _full_capacity_score(C64, v64, t, g, nbr):
    cols = np.concatenate([[t], nbr[t, :g - 1]]) if g else np.arange(C64.shape[0])
    return float(v64[cols] @ C64[t, cols])


def _literal_teacher_forced(orc, C64, v64, order, gains, eps, iters, g, nbr):
    K = len(order)
    res = orc.sgs_literal(C64, v64, K, eps, iters, g, nbr, forced=order)
    diverged, worst = 0, 0.0
    for l in range(K):
        best, picked = res["best_score"][l], res["picked_score"][l]
        scale = picked + _full_capacity_score(C64, v64, int(order[l]), g, nbr)
        if order[l] != res["best_idx"][l]:
            diverged += 1
            assert picked - best <= LIT_RTOL * scale, (
                f"step {l}: GPU picked {order[l]} (score {picked:.9g}), oracle "
                f"{res['best_idx'][l]} ({best:.9g})")
        worst = max(worst, abs(gains[l] - picked) / scale)
        assert abs(gains[l] - picked) <= LIT_RTOL * scale, (l, gains[l], picked)
    return diverged, worst


@pytest.mark.parametrize("name,N,D,K,g", [("tiny", 1024, 256, 102, 0),
                                          ("long_video", 1000, 512, 100, 0),
                                          ("short_clip", 700, 256, 70, 24)])
def test_sgs_literal_parity(orc, name, N, D, K, g):
    """Teacher-forced over every step on the GPU's own cost and capacity
    (each pick the oracle's argmin or within LIT_RTOL of its score, the
    recorded score the oracle's), the coverage objective of the kept set,
    and end to end against the oracle on its own cost and capacity
    (identical picks up to the first oracle near-tie)."""
    s = scene(name, 0, N=N, D=D)
    prm = cp.Params(g=g, sgs_mode=2)
    sel, cst = _select_case(orc, s, K, prm)
    assert cp.coverprune_check(sel["ws"]) == cp.CP_OK
    order, kept = host(sel["order"]), host(sel["kept"])
    assert np.array_equal(np.sort(order), kept) and len(set(kept.tolist())) == K
    C64 = host(cst["cost"]).astype(np.float64)
    v64 = host(cst["capacity"]).astype(np.float64)
    nbr = orc.knn_others(s["pos"], g - 1) if g else None
    div, worst = _literal_teacher_forced(orc, C64, v64, order, host(sel["gains"]), prm.sot_eps,
                                         prm.sot_iters, g, nbr)
    F = orc.objective(C64, v64, kept, 3.0, g, nbr)
    assert abs(float(host(sel["objective"])) - F) <= 1e-4 * F
    op = oracle_params(orc, cp.Params(g=g))
    pre = orc.prepare(f64(s), s["pos"], s["frame"], op)
    Co = orc.cost_matrix(f64(s), s["pos"], s["frame"], op.weights, pre["norms"])
    ora = orc.sgs_literal(Co, pre["v"], K, prm.sot_eps, prm.sot_iters, g,
                          pre["nbr"] if g else None)
    first = next((l for l in range(K) if order[l] != ora["order"][l]), K)
    if first < K:
        best, sec = ora["best_score"][first], ora["second"][first]
        t = int(ora["order"][first])
        scale = best + _full_capacity_score(Co, pre["v"], t, g, pre["nbr"] if g else None)
        assert sec - best <= LIT_RTOL * scale, (
            f"diverged at step {first} without a near-tie: best {best:.9g} second {sec:.9g}")
    jac = len(set(kept.tolist()) & set(ora["kept"].tolist())) / len(set(kept.tolist()) |
                                                                     set(ora["kept"].tolist()))
    print(f"literal {name} g={g}: teacher-forced near-ties {div}, worst score gap {worst:.3g}; "
          f"end to end equal for {first}/{K} steps, Jaccard {jac:.3f}")


@pytest.mark.parametrize("name,N,D,K,g,seed", [("long_video", 2000, 512, 200, 64, 3),
                                               ("short_clip", 1500, 256, 150, 24, 4),
                                               ("long_video", 777, 128, 60, 17, 5)])
def test_local_tiles_bounded_normaliser(orc, name, N, D, K, g, seed):
    """Local SGS (Eq. local_neighbor) with the bounded feature normaliser on
    bf16 features computes only the Morton tiles that hold a neighbour pair,
    not the all-pairs Gram.  Its lazy picks equal its full sweep bit for
    bit; teacher-forced on the dense cost of the all-pairs path (every
    greedy step, the recorded gains and the objective); end to end against
    the oracle in the same mode."""
    s = scene(name, seed, N=N, D=D)
    prm = cp.Params(g=g, norm_mode=1)
    f, pos, fr = to_dev(s)
    sel = cp.coverprune_select(f, pos, fr, K, prm)
    full = cp.coverprune_select(f, pos, fr, K, cp.Params(g=g, norm_mode=1, sgs_mode=1))
    cst = cp.coverprune_cost(f, pos, fr, prm)
    torch.cuda.synchronize()
    assert cp.coverprune_check(sel["ws"]) == cp.CP_OK
    assert cp.coverprune_check(full["ws"]) == cp.CP_OK
    for k in ("kept", "order", "gains", "objective"):
        assert torch.equal(sel[k], full[k]), k
    order, kept = host(sel["order"]), host(sel["kept"])
    nbr = orc.knn_others(s["pos"], g - 1)
    C64 = host(cst["cost"]).astype(np.float64)
    v64 = host(cst["capacity"]).astype(np.float64)
    div, _ = check_sgs_teacher_forced(orc, C64, v64, order, host(sel["gains"]),
                                      float(host(sel["objective"])), 3.0, g, nbr)
    op = oracle_params(orc, prm)
    ora = orc.select(f64(s), s["pos"], s["frame"], K, op)
    eps = measured_errors(C64, ora["C"], v64, ora["v"])
    first, jac = check_sgs_end_to_end(orc, ora, order, kept, 3.0, g, eps=eps)
    print(f"tiles {name} N={N} g={g}: teacher-forced near-ties {div}; end to end equal for "
          f"{first}/{K} steps, Jaccard {jac:.3f}")


def test_sgs_closed_forms():
    # identical tokens: dense keeps 0..K-1; local keeps {0} + {g .. g+K-2}
    N, K, g = 50, 6, 5
    f = torch.ones(N, 16, dtype=torch.bfloat16, device="cuda")
    pos = torch.zeros(N, 3, device="cuda")
    fr = torch.zeros(N, dtype=torch.int32, device="cuda")
    a = cp.coverprune_select(f, pos, fr, K, cp.Params())
    b = cp.coverprune_select(f, pos, fr, K, cp.Params(g=g))
    assert host(a["kept"]).tolist() == list(range(K))
    assert host(b["kept"]).tolist() == [0] + list(range(g, g + K - 1))
    assert abs(float(host(b["objective"])) - 3.0 * (N - g - K + 1) / N) < 1e-6
    # temporal direction: K = 1 picks the first token of frame 0
    tau = torch.tensor(np.random.default_rng(1).permutation(np.repeat(np.arange(5), 10)),
                       dtype=torch.int32, device="cuda")
    c = cp.coverprune_select(f, pos, tau, 1, cp.Params(capacity_mode=1))
    assert int(host(c["kept"])[0]) == int(np.flatnonzero(host(tau) == 0).min())


def test_sgs_deterministic_and_batched(orc):
    scs = [scene("short_clip", sd, N=700, D=256) for sd in (5, 6, 7)]
    f, pos, fr = batch_to_dev(scs)
    K = 70
    a = cp.coverprune_select(f, pos, fr, K)
    b = cp.coverprune_select(f, pos, fr, K)
    torch.cuda.synchronize()
    for k in ("kept", "order", "gains", "objective"):
        assert torch.equal(a[k], b[k]), k
    for i, s in enumerate(scs):
        one = cp.coverprune_select(*to_dev(s), K)
        for k in ("kept", "order", "gains", "objective"):
            assert torch.equal(one[k], a[k][i]), (i, k)


@pytest.mark.parametrize("g", [0, 9])
def test_sgs_batch32_launch_shape(g):
    """32 scenes in one call: the launch shape of the benchmark (several
    co-resident blocks per SM and per scene).  Every scene must equal its
    own single-scene call, whose launch shape differs."""
    scs = [scene("short_clip", sd, N=600, D=64) for sd in range(4)]
    f, pos, fr = batch_to_dev(scs * 8)
    K = 150
    prm = cp.Params(g=g)
    a = cp.coverprune_select(f, pos, fr, K, prm)
    assert cp.coverprune_check(a["ws"]) == cp.CP_OK, host(a["ws"][:32].view(torch.int32))
    singles = [cp.coverprune_select(*to_dev(s), K, prm) for s in scs]
    for b in range(32):
        for k in ("kept", "order", "gains", "objective"):
            assert torch.equal(a[k][b], singles[b % 4][k]), (b, k)


@pytest.mark.parametrize("name,N,D,K,g,B", [("tiny", 1024, 256, 102, 0, 1),
                                             ("short_clip", 1500, 512, 300, 0, 3),
                                             ("long_video", 2000, 512, 400, 20, 2),
                                             ("short_clip", 777, 128, 777, 0, 1),
                                             ("long_video", 3000, 256, 450, 0, 32),
                                             ("long_video", 2500, 256, 600, 64, 3),
                                             ("short_clip", 900, 128, 900, 12, 1),
                                             ("long_video", 1200, 64, 300, 2, 2),
                                             ("long_video", 1600, 128, 200, 0, 16)])
def test_sgs_lazy_equals_full_sweep(name, N, D, K, g, B):
    """Lazy evaluation only skips candidates whose earlier (upper-bound) gain
    cannot win, so it must reproduce the full sweep bit for bit."""
    scs = [scene(name, sd, N=N, D=D) for sd in range(min(B, 4))]
    f, pos, fr = batch_to_dev((scs * B)[:B])
    lazy = cp.coverprune_select(f, pos, fr, K, cp.Params(g=g, sgs_mode=0))
    full = cp.coverprune_select(f, pos, fr, K, cp.Params(g=g, sgs_mode=1))
    assert cp.coverprune_check(lazy["ws"]) == cp.CP_OK
    assert cp.coverprune_check(full["ws"]) == cp.CP_OK
    for k in ("kept", "order", "gains", "objective"):
        assert torch.equal(lazy[k], full[k]), k


def test_sgs_local_duplicates_equal_full_sweep():
    # coincident tokens share neighbourhoods and tie on gains: the reverse
    # lists must mark every affected candidate, and ties keep the lowest index
    rng = np.random.default_rng(7)
    base = rng.random((150, 3)).astype(np.float32) * np.float32([6, 6, 3])
    X = np.repeat(base, 4, axis=0)
    f = torch.from_numpy(np.repeat(rng.standard_normal((150, 32)).astype(np.float32), 4, axis=0))
    f = f.to(torch.bfloat16).cuda()
    pos = torch.from_numpy(X).cuda()
    fr = torch.from_numpy((np.arange(600) // 60).astype(np.int32)).cuda()
    for g in (5, 33):
        lazy = cp.coverprune_select(f, pos, fr, 200, cp.Params(g=g, sgs_mode=0))
        full = cp.coverprune_select(f, pos, fr, 200, cp.Params(g=g, sgs_mode=1))
        assert cp.coverprune_check(lazy["ws"]) == cp.CP_OK
        for k in ("kept", "order", "gains", "objective"):
            assert torch.equal(lazy[k], full[k]), (g, k)


def test_inputs_done_event_allows_overwriting_inputs():
    """cp_params.inputs_done is recorded once a call has read its inputs:
    zeroing them on another stream right after that event (while the greedy
    selection still runs) leaves every result as it was."""
    s = scene("short_clip", 0, N=2000, D=256)
    f, pos, fr = to_dev(s)
    side = torch.cuda.Stream()
    for call in ("select", "lite"):
        fn = cp.coverprune_select if call == "select" else cp.coverprune_lite_select
        ref = fn(f, pos, fr, 300)
        f2, pos2, fr2 = f.clone(), pos.clone(), fr.clone()
        ev = torch.cuda.Event()
        r = fn(f2, pos2, fr2, 300, cp.Params(inputs_done=ev))
        side.wait_event(ev)
        with torch.cuda.stream(side):
            f2.zero_()
            pos2.zero_()
            fr2.zero_()
        torch.cuda.synchronize()
        assert ev.query()
        assert torch.equal(r["kept"], ref["kept"]), call
        assert torch.equal(r["objective"], ref["objective"]), call


def test_sgs_small_edges():
    for N in (1, 2, 3):
        f = torch.randn(N, 8, device="cuda").to(torch.bfloat16)
        pos = torch.rand(N, 3, device="cuda")
        fr = torch.arange(N, dtype=torch.int32, device="cuda")
        r = cp.coverprune_select(f, pos, fr, N)
        assert host(r["kept"]).tolist() == list(range(N))
        r1 = cp.coverprune_select(f, pos, fr, 1)
        assert 0 <= int(host(r1["kept"])[0]) < N


# --------------------------------------------------------------------------
# K6-K8: Lite
# --------------------------------------------------------------------------

def _lite_check(orc, s, K, prm, dtype):
    f, pos, fr = to_dev(s)
    lt = cp.coverprune_lite_select(f, pos, fr, K, prm)
    cst = cp.coverprune_cost(f, pos, fr, prm, cost=False)
    torch.cuda.synchronize()
    vg = host(cst["capacity"])
    codes, perm = orc.morton(s["pos"], prm.voxel_m)
    b, _ = orc.lite_groups(vg, perm, K)
    np.testing.assert_array_equal(host(lt["group_start"]), b)  # exact integer grouping
    F = f64(s)
    nm = orc.normalisers(F, s["pos"], s["frame"], prm.norm_mode)
    op = oracle_params(orc, prm)
    proto, score, obj = orc.lite_select(F, s["pos"], s["frame"], op.weights, nm,
                                        vg.astype(np.float64), perm, b)
    kept = host(lt["kept"])
    group_of = np.empty(len(perm), dtype=np.int64)
    for q in range(K):
        group_of[perm[b[q]:b[q + 1]]] = q
    assert sorted(group_of[kept].tolist()) == list(range(K))  # one prototype per group
    Co = orc.cost_matrix(F, s["pos"], s["frame"], op.weights, nm)
    near = 0
    total = 0.0
    for t in kept:
        q = group_of[t]
        mem = perm[b[q]:b[q + 1]]
        sc = float(vg[mem].astype(np.float64) @ Co[t, mem])
        total += sc
        if t != proto[q]:
            near += 1
            assert sc - score[q] <= 1e-5 * max(score[q], 1e-12), (q, t, proto[q], sc, score[q])
    assert abs(float(host(lt["objective"])) - total) <= 1e-4 * total + 1e-12
    return near


@pytest.mark.parametrize("n_cap", [3, 8, 12])
@pytest.mark.parametrize("N,D,seed", [(1001, 512, 6), (4100, 1280, 7), (777, 200, 8)])
def test_capacity_from_features(orc, n_cap, N, D, seed):
    """The capacity computed from the bf16 features (Lite, and cost calls
    without the cost) at ragged N and several neighbour counts, against the
    oracle with the oracle's normalisers; Lite's capacity is the same (its
    groups equal the oracle's grouping of this capacity)."""
    s = scene("long_video", seed, N=N, D=D)
    prm = cp.Params(n_cap=n_cap)
    f, pos, fr = to_dev(s)
    out = cp.coverprune_cost(f, pos, fr, prm, cost=False)
    K = max(1, N // 10)
    lt = cp.coverprune_lite_select(f, pos, fr, K, prm)
    torch.cuda.synchronize()
    op = oracle_params(orc, prm)
    F = f64(s)
    nm = orc.normalisers(F, s["pos"], s["frame"])
    _, vo = orc.capacity(F, s["pos"], s["frame"], op.weights, nm, n_cap)
    vg = host(out["capacity"])
    assert_capacity_close(vg, vo, "bf16")
    _, perm = orc.morton(s["pos"], prm.voxel_m)
    b, _ = orc.lite_groups(vg, perm, K)
    np.testing.assert_array_equal(host(lt["group_start"]), b)


@pytest.mark.parametrize("name,N,D,K", [("tiny", 1024, 256, 102), ("long_video", 1500, 512, 150),
                                        ("short_clip", 333, 256, 100)])
def test_lite_parity(orc, name, N, D, K):
    """Teacher-forced on the GPU's capacity, then end to end against the
    oracle's Lite on its own normalisers, capacity and groups."""
    s = scene(name, 0, N=N, D=D)
    dtype = s["dtype"]
    near = _lite_check(orc, s, K, cp.Params(), dtype)
    f, pos, fr = to_dev(s)
    lt = cp.coverprune_lite_select(f, pos, fr, K)
    torch.cuda.synchronize()
    op = oracle_params(orc, cp.Params())
    ora = orc.lite(f64(s), s["pos"], s["frame"], K, op)
    moved, near_e = check_lite_end_to_end(orc, s, ora, host(lt["kept"]), host(lt["group_start"]),
                                          op.weights, dtype)
    print(f"lite {name}: near-tie prototype differences {near}/{K} forced, {near_e} end to "
          f"end, moved group starts {moved}")


@pytest.mark.parametrize("name,N,D,K", [("tiny", 1024, 256, 102), ("long_video", 1500, 512, 150)])
def test_lite_bounded_normaliser(orc, name, N, D, K):
    """Lite with the bounded feature normaliser (no Gram pass at all)."""
    s = scene(name, 2, N=N, D=D)
    near = _lite_check(orc, s, K, cp.Params(norm_mode=1), s["dtype"])
    print(f"lite bounded {name}: near-tie prototype differences {near}/{K}")


@pytest.mark.parametrize("K", [12, 25, 90])
def test_lite_group_sizes_ragged_width(orc, K):
    """Groups of ~83 members (the FMA path past 64), ~40 (several tensor-core
    tiles a group, off-diagonal tiles included) and ~11 (one diagonal tile
    fed by asynchronous copies), on a feature width that is not a multiple
    of any chunk (D = 200: the last 32-column chunk is a quarter full)."""
    s = scene("long_video", 3, N=1000, D=200)
    _lite_check(orc, s, K, cp.Params(), "bf16")
    _lite_check(orc, s, K, cp.Params(norm_mode=1), "bf16")


def test_lite_edges(orc):
    s = scene("short_clip", 4, N=200, D=64)
    _lite_check(orc, s, 1, cp.Params(), "bf16")          # one group
    _lite_check(orc, s, 200, cp.Params(), "bf16")        # every token its own group
    _lite_check(orc, s, 17, cp.Params(capacity_mode=1), "bf16")
    f, pos, fr = to_dev(s)
    lt = cp.coverprune_lite_select(f, pos, fr, 200)
    assert host(lt["kept"]).tolist() == list(range(200))


# --------------------------------------------------------------------------
# K9: gather
# --------------------------------------------------------------------------

def test_gather_byte_exact():
    scs = [scene("short_clip", sd, N=300, D=1280) for sd in (1, 2)]
    f, pos, fr = batch_to_dev(scs)
    sel = cp.coverprune_select(f, pos, fr, 40)
    fo, po, to = cp.coverprune_gather(f, pos, fr, sel["kept"])
    torch.cuda.synchronize()
    kept = host(sel["kept"])
    for b in range(2):
        np.testing.assert_array_equal(host(fo[b].view(torch.int16)),
                                      host(f[b].view(torch.int16))[kept[b]])
        np.testing.assert_array_equal(host(po[b]), host(pos[b])[kept[b]])
        np.testing.assert_array_equal(host(to[b]), host(fr[b])[kept[b]])
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    bad = sel["kept"].clone()
    bad[0, 0] = 300
    cp.coverprune_gather(f, pos, fr, bad, status=st)
    torch.cuda.synchronize()
    assert int(st) == cp.CP_EINVAL
