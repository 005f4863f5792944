"""Host-side checks of the C ABI (no GPU needed, nothing is launched).

Every call below either touches no device at all (defaults, budget,
workspace sizing, status strings) or is rejected by host-side validation
before any CUDA call is made, so these tests are safe with fake pointers.
"""
import ctypes as C
import os
import re

import pytest

import paper_2608_13226_gb300 as cp
from paper_2608_13226_gb300 import binding

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "coverprune.h")
FAKE = 0x100000  # 256-byte aligned, never dereferenced


@pytest.fixture(scope="module")
def lib():
    from paper_2608_13226_gb300 import build
    build.build()
    return cp.load()


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    names = re.findall(r"^[A-Za-z_][\w\s\*]*?\b([a-z_][a-z0-9_]*)\s*\(", src, flags=re.M)
    return sorted(set(n for n in names if n not in ("if", "while")))


def test_exports_every_declared_symbol(lib):
    names = declared_functions()
    assert len(names) >= 10
    for n in names:
        assert hasattr(lib, n), f"{n} declared in coverprune.h but not exported"
    assert sorted(binding.EXPORTS) == names


def params(**kw):
    p = binding._CpParams()
    cp.load().cp_default_params(C.byref(p))
    for k, v in kw.items():
        setattr(p, k, v)
    return p


def test_defaults(lib):
    p = params()
    assert p.struct_size == C.sizeof(binding._CpParams)
    assert (p.lambda_f, p.lambda_x, p.lambda_tau) == (1.0, 1.0, 1.0)
    assert (p.alpha_f, p.alpha_x, p.alpha_tau) == (1.0, 1.0, 1.0)
    assert p.kappa == 10.0 and p.n_cap == 8 and p.g == 0 and p.capacity_mode == 0
    assert p.sgs_mode == 0
    assert p.norm_mode == 0
    assert abs(p.sot_eps - 0.05) < 1e-7 and p.sot_iters == 20
    assert abs(p.voxel_m - 0.2) < 1e-7 and p.m0 == 0.0 and p.timeout_ms > 0
    py = cp.Params()
    for f in ("lambda_f", "kappa", "n_cap", "g", "voxel_m", "timeout_ms", "sot_eps",
              "sot_iters"):
        assert abs(getattr(py, f) - getattr(p, f)) < 1e-6


def test_budget(lib):
    # K = ceil(R N) (Sec. 3.2); the paper's efficiency run keeps 628 of 6272
    assert cp.coverprune_budget(0.1, 6272) == 628
    assert cp.coverprune_budget(0.15, 8192) == 1229
    assert [cp.coverprune_budget(r, 8192) for r in (0.05, 0.10, 0.25)] == [410, 820, 2048]
    assert cp.coverprune_budget(1.0, 17) == 17
    assert cp.coverprune_budget(1e-9, 17) == 1
    assert cp.coverprune_budget(0.0, 17) == -1
    assert cp.coverprune_budget(1.5, 17) == -1
    assert cp.coverprune_budget(0.5, 0) == -1


def test_status_strings(lib):
    for s in range(7):
        assert cp.status_string(s) and cp.status_string(s) != "unknown status"
    assert cp.status_string(99) == "unknown status"


def test_workspace_sizes(lib):
    ws = lambda op, B, N, D, K, dt=cp.CP_BF16, **kw: cp.coverprune_workspace_size(
        op, B, N, D, K, dt, cp.Params(**kw))
    a = ws(cp.CP_OP_SELECT, 1, 1000, 64, 10)
    b = ws(cp.CP_OP_SELECT, 2, 1000, 64, 10)
    assert b > a > 1000 * 1000 * 4  # holds the dense cost
    assert ws(cp.CP_OP_SELECT, 1, 1000, 64, 10, g=16) > a  # plus the local slab
    assert ws(cp.CP_OP_LITE, 1, 1000, 64, 10) < a
    assert ws(cp.CP_OP_COST, 1, 1000, 64, 0) < a
    assert ws(cp.CP_OP_KNN, 3, 1000, 8, 0) >= 256 + 3 * 64
    with pytest.raises(cp.CoverPruneError) as e:
        ws(cp.CP_OP_SELECT, 1, 20000, 64, 10)
    assert e.value.status == cp.CP_EUNSUPPORTED
    for bad in (dict(N=10, D=64, K=11), dict(N=10, D=12, K=2), dict(N=-1, D=64, K=0)):
        with pytest.raises(cp.CoverPruneError) as e:
            ws(cp.CP_OP_SELECT, 1, bad["N"], bad["D"], bad["K"])
        assert e.value.status == cp.CP_EINVAL
    with pytest.raises(cp.CoverPruneError):
        ws(cp.CP_OP_SELECT, 1, 100, 64, 10, kappa=0.0)
    with pytest.raises(cp.CoverPruneError):
        ws(cp.CP_OP_SELECT, 1, 100, 64, 10, lambda_f=float("nan"))


def _select(lib, p, B=1, N=100, D=64, K=10, dt=cp.CP_BF16, feats=FAKE, kept=FAKE, ws=FAKE,
            ws_bytes=1 << 40):
    return lib.coverprune_select(C.c_void_p(feats), dt, C.c_void_p(FAKE), C.c_void_p(FAKE), B, N,
                                 D, K, C.byref(p), C.c_void_p(kept), None, None, None,
                                 C.c_void_p(ws), ws_bytes, None)


def test_validation_rejects_before_launch(lib):
    p = params()
    assert _select(lib, p, K=101) == cp.CP_EINVAL           # K > N
    assert _select(lib, p, K=-1) == cp.CP_EINVAL
    assert _select(lib, p, D=12) == cp.CP_EINVAL            # bf16 rows need D % 8 == 0
    assert _select(lib, p, D=6, dt=cp.CP_F32) == cp.CP_EINVAL
    assert _select(lib, p, dt=7) == cp.CP_EINVAL
    assert _select(lib, p, feats=0) == cp.CP_EINVAL          # NULL input
    assert _select(lib, p, feats=FAKE + 8) == cp.CP_EINVAL   # misaligned features
    assert _select(lib, p, kept=0) == cp.CP_EINVAL           # NULL output
    assert _select(lib, p, ws=0) == cp.CP_EWORKSPACE
    assert _select(lib, p, ws=FAKE + 64) == cp.CP_EWORKSPACE  # misaligned workspace
    assert _select(lib, p, ws_bytes=1024) == cp.CP_EWORKSPACE
    assert _select(lib, p, N=20000, K=10) == cp.CP_EUNSUPPORTED
    assert _select(lib, params(struct_size=4)) == cp.CP_EINVAL
    assert _select(lib, params(kappa=-1.0)) == cp.CP_EINVAL
    assert _select(lib, params(capacity_mode=2)) == cp.CP_EINVAL
    assert _select(lib, params(timeout_ms=0.0)) == cp.CP_EINVAL
    assert _select(lib, params(sgs_mode=3)) == cp.CP_EINVAL
    assert _select(lib, params(sgs_mode=-1)) == cp.CP_EINVAL
    assert _select(lib, params(sgs_mode=2, sot_eps=0.0)) == cp.CP_EINVAL
    assert _select(lib, params(sgs_mode=2, sot_eps=float("nan"))) == cp.CP_EINVAL
    assert _select(lib, params(sgs_mode=2, sot_iters=0)) == cp.CP_EINVAL
    assert _select(lib, params(sgs_mode=2, sot_iters=10001)) == cp.CP_EINVAL
    assert _select(lib, params(norm_mode=2)) == cp.CP_EINVAL
    assert _select(lib, params(norm_mode=-1)) == cp.CP_EINVAL
    assert _select(lib, params(lambda_x=float("inf"))) == cp.CP_EINVAL
    # empty problems are no-ops
    assert _select(lib, p, B=0) == cp.CP_OK
    assert _select(lib, p, N=0, K=0) == cp.CP_OK
    assert _select(lib, p, K=0) == cp.CP_OK


def test_other_entry_points_validate(lib):
    p = params()
    P = lambda x: C.c_void_p(x)
    assert lib.coverprune_lite_select(P(FAKE), 1, P(FAKE), P(FAKE), 1, 100, 64, 101, C.byref(p),
                                      P(FAKE), None, None, P(FAKE), 1 << 40, None) == cp.CP_EINVAL
    assert lib.coverprune_lite_select(P(FAKE), 1, P(FAKE), P(FAKE), 1, 100, 64, 10, C.byref(p),
                                      P(FAKE), None, None, P(FAKE), 16, None) == cp.CP_EWORKSPACE
    assert lib.coverprune_cost(P(FAKE), 1, P(FAKE), P(FAKE), 1, 100, 60, C.byref(p), P(FAKE),
                               None, None, P(FAKE), 1 << 40, None) == cp.CP_EINVAL
    assert lib.coverprune_cost(P(FAKE), 1, P(FAKE), P(FAKE), 1, 100, 64, C.byref(p), P(FAKE + 2),
                               None, None, P(FAKE), 1 << 40, None) == cp.CP_EINVAL
    assert lib.coverprune_knn(P(FAKE), 1, 10, 10, P(FAKE), None, P(FAKE), 1 << 20,
                              None) == cp.CP_EINVAL  # k > N - 1
    assert lib.coverprune_knn(P(FAKE), 1, 10, 3, P(FAKE), None, P(FAKE), 8,
                              None) == cp.CP_EWORKSPACE
    assert lib.coverprune_gather(P(FAKE), 1, P(FAKE), P(FAKE), 1, 100, 64, P(FAKE), 101, P(FAKE),
                                 None, None, None, None) == cp.CP_EINVAL
    assert lib.coverprune_gather(P(FAKE), 1, P(FAKE), P(FAKE), 1, 100, 64, P(FAKE), 5, P(FAKE + 4),
                                 None, None, None, None) == cp.CP_EINVAL
    assert lib.coverprune_gather(P(FAKE), 1, None, P(FAKE), 1, 100, 64, P(FAKE), 5, P(FAKE),
                                 P(FAKE), None, None, None) == cp.CP_EINVAL  # pos_out w/o pos
    assert lib.coverprune_barrier_selftest(2, 3, 10.0, P(FAKE), 16, None) == cp.CP_EWORKSPACE
    assert lib.coverprune_barrier_selftest(0, 3, 10.0, P(FAKE), 256, None) == cp.CP_EINVAL
    assert lib.coverprune_barrier_selftest(2, 3, -1.0, P(FAKE), 256, None) == cp.CP_EINVAL
    assert lib.coverprune_check(None, None) == cp.CP_EINVAL


def test_binding_refuses_cpu_tensors(lib):
    import torch
    f = torch.zeros(10, 8, dtype=torch.bfloat16)
    x = torch.zeros(10, 3)
    t = torch.zeros(10, dtype=torch.int32)
    with pytest.raises(ValueError):
        cp.coverprune_select(f, x, t, 2)
    with pytest.raises(ValueError):
        cp.coverprune_cost(f, x, t)
