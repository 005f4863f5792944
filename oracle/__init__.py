"""CoverPrune CPU oracle -- TEST INFRASTRUCTURE, not part of the product.

A ctypes front end for ``coverprune_oracle.c``: a plain, slow, scalar fp64
restatement of the FST cost (Sec. 3.3, Eqs. fst_metrics / fst_cost), the FST
capacity (Sec. 3.4, Eqs. fst_capacity_score / fst_capacity), Spatial-Guided
Greedy Selection (Sec. 3.5, Eqs. srpot, local_neighbor, greedy_flow,
sgs_select, sgs_update) and CoverPrune-Lite (Sec. 4, Eqs. lite_group,
lite_select, blk_plan, blk_ot).

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline
and reference legs may import this package.  It shares no code with the CUDA
library and imports nothing from it; inputs come from the seeded scene
generator, which holds none of the method's arithmetic.

Every function here marshals numpy arrays and calls the C code; no arithmetic
of the method happens in Python except the end-to-end drivers
(:func:`select`, :func:`lite`), which only chain the C steps in the paper's
order.

Parity unpinned: none -- every function is pinned by the ``-m "not gpu"``
tests (worked example, closed forms, exhaustive search, LP optimality of the
objective, library routines).
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "coverprune_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libcoverprune_oracle.so")
_lock = threading.Lock()
_lib = None

GCC_FLAGS = ["-O2", "-std=gnu11", "-fopenmp", "-ffp-contract=off", "-fPIC", "-shared",
             "-Wall", "-Wextra"]


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (fp contraction off) into oracle/_build."""
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    subprocess.run(["gcc", *GCC_FLAGS, "-o", tmp, _SRC, "-lm"], check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class _Weights(C.Structure):
    _fields_ = [(n, C.c_double) for n in
                ("lambda_f", "lambda_x", "lambda_tau", "kappa", "alpha_f", "alpha_x",
                 "alpha_tau")]


class _Norms(C.Structure):
    _fields_ = [(n, C.c_double) for n in
                ("f_lo", "f_hi", "x_lo", "x_hi", "tau_lo", "tau_hi")]


@dataclass
class Weights:
    """Weights of Eq. fst_cost (lambda, kappa) and Eq. fst_capacity_score
    (alpha).  Defaults: lambda = alpha = 1 (Sec. 5.1 implementation details);
    kappa = 10 (the paper gives no value)."""
    lambda_f: float = 1.0
    lambda_x: float = 1.0
    lambda_tau: float = 1.0
    kappa: float = 10.0
    alpha_f: float = 1.0
    alpha_x: float = 1.0
    alpha_tau: float = 1.0

    def _c(self) -> _Weights:
        return _Weights(self.lambda_f, self.lambda_x, self.lambda_tau, self.kappa,
                        self.alpha_f, self.alpha_x, self.alpha_tau)


@dataclass
class Norms:
    """Per-scene min-max ranges of d_f, d_x and d_tau (Sec. 3.3)."""
    f_lo: float
    f_hi: float
    x_lo: float
    x_hi: float
    tau_lo: float
    tau_hi: float

    def _c(self) -> _Norms:
        return _Norms(self.f_lo, self.f_hi, self.x_lo, self.x_hi, self.tau_lo, self.tau_hi)


_P = C.c_void_p
_I64 = C.c_int64


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = C.CDLL(build())
        lib.orc_set_threads.argtypes = [C.c_int]
        lib.orc_get_threads.restype = C.c_int
        lib.orc_normalisers.argtypes = [_I64, _I64, _P, _P, _P, C.POINTER(_Norms)]
        lib.orc_normalisers_mode.argtypes = [_I64, _I64, _P, _P, _P, C.c_int,
                                             C.POINTER(_Norms)]
        lib.orc_cost_rows.argtypes = [_I64, _I64, _P, _P, _P, C.POINTER(_Weights),
                                      C.POINTER(_Norms), _I64, _I64, _P]
        lib.orc_cost_pairs.argtypes = [_I64, _I64, _P, _P, _P, C.POINTER(_Weights),
                                       C.POINTER(_Norms), _I64, _P, _P, _P]
        lib.orc_knn_others.argtypes = [_I64, _P, _I64, _P]
        lib.orc_capacity.argtypes = [_I64, _I64, _P, _P, _P, C.POINTER(_Weights),
                                     C.POINTER(_Norms), _I64, _P, C.c_int, _P, _P]
        lib.orc_objective.argtypes = [_I64, _P, _P, _I64, _P, C.c_double, _I64, _P, _P]
        lib.orc_sgs.argtypes = [_I64, _P, _P, _I64, _P, _I64, C.c_double, _P, _P, _P,
                                _P, _P, _P, _P]
        lib.orc_morton.argtypes = [_I64, _P, C.c_float, _P, _P]
        lib.orc_lite_groups.argtypes = [_I64, _I64, _P, _P, _P, _P]
        lib.orc_lite_select.argtypes = [_I64, _I64, _P, _P, _P, C.POINTER(_Weights),
                                        C.POINTER(_Norms), _P, _P, _P, _I64, _P, _P, _P]
        lib.orc_sot_sinkhorn.argtypes = [_I64, _I64, _P, _P, _P, C.c_double, _I64, _P, _P, _P,
                                         _P]
        lib.orc_sgs_literal.argtypes = [_I64, _P, _P, _I64, _P, _I64, C.c_double, _I64, _P, _P,
                                        _P, _P, _P, _P]
        for fn in ("orc_normalisers", "orc_normalisers_mode", "orc_cost_rows", "orc_cost_pairs", "orc_knn_others",
                   "orc_capacity", "orc_objective", "orc_sgs", "orc_morton",
                   "orc_lite_groups", "orc_lite_select", "orc_sot_sinkhorn",
                   "orc_sgs_literal"):
            getattr(lib, fn).restype = C.c_int
        _lib = lib
        return lib


def _ptr(a: np.ndarray | None):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


def _check(rc: int, what: str):
    if rc != 0:
        raise ValueError(f"oracle {what} failed with code {rc}")


def _f64(F) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(F, dtype=np.float64))


def _pos(X) -> np.ndarray:
    X = np.ascontiguousarray(np.asarray(X, dtype=np.float32))
    assert X.ndim == 2 and X.shape[1] == 3
    return X


def _tau(t) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(t, dtype=np.int32))


def set_threads(n: int) -> None:
    _load().orc_set_threads(int(n))


def get_threads() -> int:
    return int(_load().orc_get_threads())


# --------------------------------------------------------------------------
# Cost and capacity
# --------------------------------------------------------------------------

def normalisers(F, X, tau, norm_mode: int = 0) -> Norms:
    """Min and max of d_f, d_x, d_tau over all ordered pairs (Sec. 3.3);
    norm_mode 1 takes the bounds [0, 2] of d_f = 1 - cos instead of its
    measured range (the bounded feature normaliser)."""
    F, X, tau = _f64(F), _pos(X), _tau(tau)
    N, D = F.shape
    out = _Norms()
    _check(_load().orc_normalisers_mode(N, D, _ptr(F), _ptr(X), _ptr(tau), int(norm_mode),
                                        C.byref(out)), "normalisers")
    return Norms(out.f_lo, out.f_hi, out.x_lo, out.x_hi, out.tau_lo, out.tau_hi)


def cost_rows(F, X, tau, w: Weights, nm: Norms, s0: int, s1: int) -> np.ndarray:
    """Rows [s0, s1) of the FST cost C (Eq. fst_cost), row = source token."""
    F, X, tau = _f64(F), _pos(X), _tau(tau)
    N, D = F.shape
    out = np.empty((s1 - s0, N), dtype=np.float64)
    wc, nc = w._c(), nm._c()
    _check(_load().orc_cost_rows(N, D, _ptr(F), _ptr(X), _ptr(tau), C.byref(wc),
                                 C.byref(nc), s0, s1, _ptr(out)), "cost_rows")
    return out


def cost_matrix(F, X, tau, w: Weights, nm: Norms) -> np.ndarray:
    return cost_rows(F, X, tau, w, nm, 0, np.asarray(F).shape[0])


def cost_pairs(F, X, tau, w: Weights, nm: Norms, S, T) -> np.ndarray:
    """C(S[p], T[p]) for sampled pairs."""
    F, X, tau = _f64(F), _pos(X), _tau(tau)
    N, D = F.shape
    S = np.ascontiguousarray(np.asarray(S, dtype=np.int64))
    T = np.ascontiguousarray(np.asarray(T, dtype=np.int64))
    out = np.empty(S.shape[0], dtype=np.float64)
    wc, nc = w._c(), nm._c()
    _check(_load().orc_cost_pairs(N, D, _ptr(F), _ptr(X), _ptr(tau), C.byref(wc),
                                  C.byref(nc), S.shape[0], _ptr(S), _ptr(T), _ptr(out)),
           "cost_pairs")
    return out


def knn_others(X, k: int) -> np.ndarray:
    """[N, k] nearest other tokens in 3D, ordered by (fp32 d^2, index)."""
    X = _pos(X)
    N = X.shape[0]
    out = np.empty((N, max(k, 0)), dtype=np.int32)
    _check(_load().orc_knn_others(N, _ptr(X), k, _ptr(out)), "knn_others")
    return out


def capacity(F, X, tau, w: Weights, nm: Norms, n: int, nbr=None, mode: int = 0):
    """(r, v) of Eqs. fst_capacity_score / fst_capacity.  nbr defaults to the
    n nearest others; n is clamped to N-1."""
    F, X, tau = _f64(F), _pos(X), _tau(tau)
    N, D = F.shape
    n = min(n, N - 1)
    if nbr is None:
        nbr = knn_others(X, n)
    nbr = np.ascontiguousarray(np.asarray(nbr, dtype=np.int32)[:, :n])
    r = np.empty(N, dtype=np.float64)
    v = np.empty(N, dtype=np.float64)
    wc, nc = w._c(), nm._c()
    _check(_load().orc_capacity(N, D, _ptr(F), _ptr(X), _ptr(tau), C.byref(wc),
                                C.byref(nc), n, _ptr(nbr), mode, _ptr(r), _ptr(v)),
           "capacity")
    return r, v


# --------------------------------------------------------------------------
# SGS
# --------------------------------------------------------------------------

def _nbr_g(nbr_g, N, g):
    """(neighbour lists [N, g-1] or None, g): g <= 0 or g >= N (or no lists
    given) means every token; g = 1 means the token alone."""
    if g <= 0 or g >= N or (nbr_g is None and g != 1):
        return None, N
    if g == 1:
        return None, 1
    return np.ascontiguousarray(np.asarray(nbr_g, dtype=np.int32)[:, :g - 1]), g


def objective(Cm, v, S, M0: float, g: int = 0, nbr_g=None) -> float:
    """F_g(S) = sum_j v_j min(M0, min_{s in S, j in M_g(s)} C(s, j))."""
    Cm = _f64(Cm)
    v = _f64(v)
    N = Cm.shape[0]
    nb, g = _nbr_g(nbr_g, N, g)
    S = np.ascontiguousarray(np.asarray(S, dtype=np.int64))
    out = C.c_double()
    _check(_load().orc_objective(N, _ptr(Cm), _ptr(v), g, _ptr(nb), M0, S.shape[0],
                                 _ptr(S), C.byref(out)), "objective")
    return float(out.value)


def sgs(Cm, v, K: int, M0: float, g: int = 0, nbr_g=None, forced=None) -> dict:
    """K greedy steps (Sec. 3.5) on cost matrix Cm [N, N] (row = source).

    Returns order, best_idx, best_gain, second, picked_gain, F_after (per
    step), kept (ascending) and F (final objective).  With ``forced`` the
    oracle adds forced[l] at step l but still reports its own argmax."""
    Cm = _f64(Cm)
    v = _f64(v)
    N = Cm.shape[0]
    nb, g = _nbr_g(nbr_g, N, g)
    fo = None if forced is None else np.ascontiguousarray(np.asarray(forced, dtype=np.int64))
    res = {k: np.empty(K, dtype=np.int64) for k in ("order", "best_idx")}
    res.update({k: np.empty(K, dtype=np.float64) for k in
                ("best_gain", "second", "picked_gain", "F_after")})
    _check(_load().orc_sgs(N, _ptr(Cm), _ptr(v), g, _ptr(nb), K, M0, _ptr(fo),
                           _ptr(res["order"]), _ptr(res["best_idx"]),
                           _ptr(res["best_gain"]), _ptr(res["second"]),
                           _ptr(res["picked_gain"]), _ptr(res["F_after"])), "sgs")
    res["kept"] = np.sort(res["order"])
    res["F"] = float(res["F_after"][-1]) if K > 0 else float(M0 * v.sum())
    return res


def sot_sinkhorn(Crows, u, v, eps: float, iters: int, g0=None) -> dict:
    """Entropic semi-relaxed OT (Eq. srpot_sinkhorn) between the sources of
    the rows of Crows [m, N] (masses u) and N targets (capacities v), by
    `iters` dual block-coordinate iterations from target potentials g0
    (zeros by default).  Returns f [m], g [N], colsum = P^T 1 [N], P [m, N]."""
    Crows = np.ascontiguousarray(np.asarray(Crows, dtype=np.float64))
    m, N = Crows.shape
    u, v = _f64(u), _f64(v)
    g = np.zeros(N) if g0 is None else np.array(g0, dtype=np.float64)
    f = np.empty(max(m, 1))
    col = np.empty(N)
    P = np.empty((m, N))
    _check(_load().orc_sot_sinkhorn(m, N, _ptr(Crows), _ptr(u), _ptr(v), float(eps), int(iters),
                                    _ptr(f), _ptr(g), _ptr(col), _ptr(P)), "sot_sinkhorn")
    return {"f": f[:m], "g": g, "colsum": col, "P": P}


def sgs_literal(Cm, v, K: int, eps: float, iters: int, g: int = 0, nbr_g=None,
                forced=None) -> dict:
    """K steps of SGS as Eqs. greedy_flow / sgs_select print it: residual
    capacity r = [v - P^T 1]_+ of the entropic semi-relaxed OT from the
    selected tokens (mass 1/K each), next token = argmin over unselected t
    of sum_{j in M_g(t)} r_j C(t, j) (lowest index on exact ties).

    Returns order, best_idx, best_score, second, picked_score (per step) and
    kept (ascending).  With ``forced`` the oracle adds forced[l] at step l
    but still reports its own argmin."""
    Cm = _f64(Cm)
    v = _f64(v)
    N = Cm.shape[0]
    nb, g = _nbr_g(nbr_g, N, g)
    fo = None if forced is None else np.ascontiguousarray(np.asarray(forced, dtype=np.int64))
    res = {k: np.empty(K, dtype=np.int64) for k in ("order", "best_idx")}
    res.update({k: np.empty(K, dtype=np.float64) for k in
                ("best_score", "second", "picked_score")})
    _check(_load().orc_sgs_literal(N, _ptr(Cm), _ptr(v), g, _ptr(nb), K, float(eps), int(iters),
                                   _ptr(fo), _ptr(res["order"]), _ptr(res["best_idx"]),
                                   _ptr(res["best_score"]), _ptr(res["second"]),
                                   _ptr(res["picked_score"])), "sgs_literal")
    res["kept"] = np.sort(res["order"])
    return res


# --------------------------------------------------------------------------
# Lite
# --------------------------------------------------------------------------

def morton(X, voxel: float):
    """(codes uint32 [N], perm int64 [N]): Morton order of Sec. 4.1."""
    X = _pos(X)
    N = X.shape[0]
    codes = np.empty(N, dtype=np.uint32)
    perm = np.empty(N, dtype=np.int64)
    _check(_load().orc_morton(N, _ptr(X), C.c_float(voxel), _ptr(codes), _ptr(perm)),
           "morton")
    return codes, perm


def lite_groups(v, perm, K: int):
    """(b int64 [K+1], Q uint64 [N]): capacity-guided groups of Eq. lite_group."""
    v32 = np.ascontiguousarray(np.asarray(v, dtype=np.float32))
    perm = np.ascontiguousarray(np.asarray(perm, dtype=np.int64))
    N = v32.shape[0]
    b = np.empty(K + 1, dtype=np.int64)
    Q = np.empty(N, dtype=np.uint64)
    _check(_load().orc_lite_groups(N, K, _ptr(v32), _ptr(perm), _ptr(b), _ptr(Q)),
           "lite_groups")
    return b, Q


def lite_select(F, X, tau, w: Weights, nm: Norms, v, perm, b):
    """(proto [K], score [K], objective): Eq. lite_select per group."""
    F, X, tau = _f64(F), _pos(X), _tau(tau)
    N, D = F.shape
    v = _f64(v)
    perm = np.ascontiguousarray(np.asarray(perm, dtype=np.int64))
    b = np.ascontiguousarray(np.asarray(b, dtype=np.int64))
    K = b.shape[0] - 1
    proto = np.empty(K, dtype=np.int64)
    score = np.empty(K, dtype=np.float64)
    obj = C.c_double()
    wc, nc = w._c(), nm._c()
    _check(_load().orc_lite_select(N, D, _ptr(F), _ptr(X), _ptr(tau), C.byref(wc),
                                   C.byref(nc), _ptr(v), _ptr(perm), _ptr(b), K,
                                   _ptr(proto), _ptr(score), C.byref(obj)), "lite_select")
    return proto, score, float(obj.value)


# --------------------------------------------------------------------------
# End-to-end drivers (the paper's order of steps, nothing more)
# --------------------------------------------------------------------------

@dataclass
class Params:
    """Method parameters.  n_cap = |N_n| (capacity neighbours), g = |M_g|
    (0 = all tokens), capacity_mode 0 = FST capacity, 1 = uniform,
    m0 = initial coverage cost (<= 0 means lambda_f + lambda_x + lambda_tau),
    voxel = Morton cell in metres, norm_mode 0 = min-max feature normaliser,
    1 = bounded (d_f / 2)."""
    weights: Weights = None
    n_cap: int = 8
    g: int = 0
    capacity_mode: int = 0
    m0: float = 0.0
    voxel: float = 0.2
    norm_mode: int = 0

    def __post_init__(self):
        if self.weights is None:
            self.weights = Weights()

    def M0(self) -> float:
        w = self.weights
        return self.m0 if self.m0 > 0 else w.lambda_f + w.lambda_x + w.lambda_tau


def prepare(F, X, tau, prm: Params) -> dict:
    """Normalisers, capacity neighbours and capacity of one scene."""
    N = np.asarray(F).shape[0]
    nm = normalisers(F, X, tau, prm.norm_mode)
    n = min(prm.n_cap, N - 1)
    g = prm.g if 0 < prm.g < N else N
    k = max(n, g - 1) if g < N else n
    nbr = knn_others(X, k)
    r, v = capacity(F, X, tau, prm.weights, nm, n, nbr[:, :n], prm.capacity_mode)
    return {"norms": nm, "nbr": nbr, "n": n, "g": g, "r": r, "v": v}


def select(F, X, tau, K: int, prm: Params) -> dict:
    """Full CoverPrune on one scene: cost, capacity, SGS (Sec. 3.3-3.5)."""
    pre = prepare(F, X, tau, prm)
    Cm = cost_matrix(F, X, tau, prm.weights, pre["norms"])
    nb = pre["nbr"] if pre["g"] < Cm.shape[0] else None
    res = sgs(Cm, pre["v"], K, prm.M0(), pre["g"], nb)
    res.update(pre)
    res["C"] = Cm
    return res


def lite(F, X, tau, K: int, prm: Params) -> dict:
    """CoverPrune-Lite on one scene (Sec. 4.1)."""
    pre = prepare(F, X, tau, prm)
    codes, perm = morton(X, prm.voxel)
    b, Q = lite_groups(pre["v"], perm, K)
    proto, score, obj = lite_select(F, X, tau, prm.weights, pre["norms"], pre["v"], perm, b)
    pre.update({"codes": codes, "perm": perm, "b": b, "Q": Q, "proto": proto,
                "score": score, "objective": obj, "kept": np.sort(proto)})
    return pre
