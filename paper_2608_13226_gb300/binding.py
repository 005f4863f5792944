"""Thin ctypes binding over libcoverprune.so (include/coverprune.h).

Argument marshalling only: every step of the CoverPrune path runs in the CUDA
library.  Tensors must be CUDA tensors; PyTorch provides device memory and the
current stream.  There is no CPU fallback: if the library is missing, loading
fails with an error.
"""
from __future__ import annotations

import ctypes as C
import os
import threading
from dataclasses import dataclass, fields

import torch

from . import build as _build

CP_OK, CP_EINVAL, CP_EWORKSPACE, CP_ECUDA, CP_ETIMEOUT, CP_EUNSUPPORTED, CP_EDEVICE = range(7)
CP_F32, CP_BF16 = 0, 1
CP_OP_COST, CP_OP_SELECT, CP_OP_LITE, CP_OP_KNN = 0, 1, 2, 3

# every symbol declared in include/coverprune.h
EXPORTS = ("cp_default_params", "coverprune_budget", "coverprune_workspace_size",
           "coverprune_status_string", "coverprune_check", "coverprune_cost",
           "coverprune_select", "coverprune_lite_select", "coverprune_knn",
           "coverprune_knn_noalloc",
           "coverprune_gather", "coverprune_barrier_selftest", "coverprune_profile_enable",
           "coverprune_profile_read", "coverprune_last_error", "coverprune_call_stats",
           "coverprune_version")
STAGES = ("prep", "gram", "cost", "capacity", "sgs", "lite_order", "lite_proto", "output",
          "slab")


class CoverPruneError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        msg = f"{what}: {status_string(status)} (status {status})"
        if status == CP_ECUDA:
            msg += f": {_lib().coverprune_last_error().decode()}"
        super().__init__(msg)


class _CpParams(C.Structure):
    _fields_ = [("struct_size", C.c_uint32),
                ("lambda_f", C.c_float), ("lambda_x", C.c_float), ("lambda_tau", C.c_float),
                ("kappa", C.c_float),
                ("alpha_f", C.c_float), ("alpha_x", C.c_float), ("alpha_tau", C.c_float),
                ("n_cap", C.c_int32), ("g", C.c_int32), ("capacity_mode", C.c_int32),
                ("voxel_m", C.c_float), ("m0", C.c_float), ("timeout_ms", C.c_float),
                ("sgs_mode", C.c_int32), ("norm_mode", C.c_int32),
                ("sot_eps", C.c_float), ("sot_iters", C.c_int32),
                ("inputs_done", C.c_void_p)]


class _CallStats(C.Structure):
    _fields_ = [("gain_evaluations", C.c_uint64), ("rounds", C.c_uint64),
                ("cost_bytes_read", C.c_uint64)]


@dataclass
class Params:
    """Mirror of cp_params (see include/coverprune.h for the meaning of each
    field).  Defaults match cp_default_params."""
    lambda_f: float = 1.0
    lambda_x: float = 1.0
    lambda_tau: float = 1.0
    kappa: float = 10.0
    alpha_f: float = 1.0
    alpha_x: float = 1.0
    alpha_tau: float = 1.0
    n_cap: int = 8
    g: int = 0
    capacity_mode: int = 0
    voxel_m: float = 0.2
    m0: float = 0.0
    timeout_ms: float = 2000.0
    sgs_mode: int = 0
    norm_mode: int = 0
    sot_eps: float = 0.05
    sot_iters: int = 20
    # not a method parameter: a torch.cuda.Event the call records once it has
    # read the last of its inputs (cp_params.inputs_done), or None
    inputs_done: object = None

    def _c(self) -> _CpParams:
        p = _CpParams()
        _lib().cp_default_params(C.byref(p))
        for f in fields(self):
            if f.name == "inputs_done":
                ev = self.inputs_done
                if ev is not None and not ev.cuda_event:
                    ev.record()  # torch creates its CUDA event on first record
                p.inputs_done = None if ev is None else C.c_void_p(ev.cuda_event)
            else:
                setattr(p, f.name, getattr(self, f.name))
        return p


_lock = threading.Lock()
_L = None


def library_path() -> str:
    return _build.LIB


def _lib():
    global _L
    if _L is not None:
        return _L
    with _lock:
        if _L is not None:
            return _L
        path = _build.LIB
        if not os.path.exists(path):
            raise RuntimeError(
                f"CoverPrune CUDA library not found at {path}; build it with "
                "paper_2608_13226_gb300.build.build() (there is no CPU fallback)")
        lib = C.CDLL(path)
        P, I64, I32, SZ = C.c_void_p, C.c_int64, C.c_int, C.c_size_t
        PP = C.POINTER(_CpParams)
        lib.cp_default_params.argtypes = [PP]
        lib.cp_default_params.restype = None
        lib.coverprune_budget.argtypes = [C.c_double, I64]
        lib.coverprune_budget.restype = I64
        lib.coverprune_workspace_size.argtypes = [I32, I64, I64, I64, I64, I32, PP,
                                                  C.POINTER(C.c_size_t)]
        lib.coverprune_status_string.argtypes = [I32]
        lib.coverprune_status_string.restype = C.c_char_p
        lib.coverprune_check.argtypes = [P, P]
        lib.coverprune_cost.argtypes = [P, I32, P, P, I64, I64, I64, PP, P, P, P, P, SZ, P]
        lib.coverprune_select.argtypes = [P, I32, P, P, I64, I64, I64, I64, PP, P, P, P, P, P,
                                          SZ, P]
        lib.coverprune_lite_select.argtypes = [P, I32, P, P, I64, I64, I64, I64, PP, P, P, P, P,
                                               SZ, P]
        lib.coverprune_knn.argtypes = [P, I64, I64, I64, P, P, P, SZ, P]
        lib.coverprune_knn_noalloc.argtypes = [P, I64, I64, I64, P, P, P]
        lib.coverprune_gather.argtypes = [P, I32, P, P, I64, I64, I64, P, I64, P, P, P, P, P]
        lib.coverprune_barrier_selftest.argtypes = [C.c_int32, C.c_int32, C.c_float, P, SZ, P]
        lib.coverprune_call_stats.argtypes = [P, P, C.POINTER(_CallStats)]
        lib.coverprune_last_error.argtypes = []
        lib.coverprune_last_error.restype = C.c_char_p
        lib.coverprune_profile_enable.argtypes = [I32]
        lib.coverprune_profile_read.argtypes = [P, P, I32]
        for fn in EXPORTS:
            if fn not in ("cp_default_params", "coverprune_budget", "coverprune_status_string",
                          "coverprune_last_error"):
                getattr(lib, fn).restype = I32
        _L = lib
        return lib


def load():
    """Load the library (raises if it is missing)."""
    return _lib()


def status_string(status: int) -> str:
    return _lib().coverprune_status_string(int(status)).decode()


def _check(st: int, what: str):
    if st != CP_OK:
        raise CoverPruneError(st, what)


def _ptr(t):
    return None if t is None else C.c_void_p(t.data_ptr())


def _stream():
    return C.c_void_p(torch.cuda.current_stream().cuda_stream)


def _dtype(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return CP_BF16
    if t.dtype == torch.float32:
        return CP_F32
    raise TypeError(f"features must be bfloat16 or float32, got {t.dtype}")


def _batched(feats, pos, frame):
    if feats.dim() == 2:
        feats, pos, frame = feats.unsqueeze(0), pos.unsqueeze(0), frame.unsqueeze(0)
    for name, t in (("feats", feats), ("pos", pos), ("frame", frame)):
        if not t.is_cuda:
            raise ValueError(f"{name} must be a CUDA tensor")
        if not t.is_contiguous():
            raise ValueError(f"{name} must be contiguous")
    if pos.dtype != torch.float32 or frame.dtype != torch.int32:
        raise TypeError("pos must be float32 and frame int32")
    B, N, D = feats.shape
    if tuple(pos.shape) != (B, N, 3) or tuple(frame.shape) != (B, N):
        raise ValueError("shapes must be feats [B,N,D], pos [B,N,3], frame [B,N]")
    return feats, pos, frame, B, N, D


def coverprune_budget(R: float, N: int) -> int:
    return int(_lib().coverprune_budget(float(R), int(N)))


def coverprune_workspace_size(op: int, B: int, N: int, D: int, K: int, dtype: int,
                              params: Params | None = None) -> int:
    p = (params or Params())._c()
    out = C.c_size_t()
    _check(_lib().coverprune_workspace_size(op, B, N, D, K, dtype, C.byref(p), C.byref(out)),
           "coverprune_workspace_size")
    return int(out.value)


def workspace(op: int, B: int, N: int, D: int, K: int, dtype: int,
              params: Params | None = None, device=None) -> torch.Tensor:
    n = coverprune_workspace_size(op, B, N, D, K, dtype, params)
    return torch.empty(max(n, 256), dtype=torch.uint8, device=device or "cuda")


def _ws(ws, op, B, N, D, K, dt, params, device):
    if ws is None:
        ws = workspace(op, B, N, D, K, dt, params, device)
    if ws.data_ptr() % 256:
        raise ValueError("workspace must be 256-byte aligned")
    return ws


def coverprune_check(ws: torch.Tensor) -> int:
    """Synchronise the current stream and return the device status word."""
    return int(_lib().coverprune_check(_ptr(ws), _stream()))


def coverprune_cost(feats, pos, frame, params: Params | None = None, *, cost=True,
                    capacity=True, norms=True, ws=None, out=None) -> dict:
    """FST cost [B,N,N], capacity [B,N] and normalisers [B,6] (or [N,N]... for
    unbatched input).  ``out`` may supply preallocated output tensors."""
    unbatched = feats.dim() == 2
    feats, pos, frame, B, N, D = _batched(feats, pos, frame)
    dt = _dtype(feats)
    params = params or Params()
    out = dict(out or {})
    dev = feats.device
    if cost and "cost" not in out:
        out["cost"] = torch.empty(B, N, N, dtype=torch.float32, device=dev)
    if capacity and "capacity" not in out:
        out["capacity"] = torch.empty(B, N, dtype=torch.float32, device=dev)
    if norms and "norms" not in out:
        out["norms"] = torch.empty(B, 6, dtype=torch.float32, device=dev)
    ws = _ws(ws, CP_OP_COST, B, N, D, 0, dt, params, dev)
    p = params._c()
    _check(_lib().coverprune_cost(_ptr(feats), dt, _ptr(pos), _ptr(frame), B, N, D, C.byref(p),
                                  _ptr(out.get("cost")), _ptr(out.get("capacity")),
                                  _ptr(out.get("norms")), _ptr(ws), ws.numel(), _stream()),
           "coverprune_cost")
    if unbatched:
        out = {k: v[0] for k, v in out.items()}
    out["ws"] = ws
    return out


def coverprune_select(feats, pos, frame, K: int, params: Params | None = None, *, order=True,
                      gains=True, objective=True, ws=None, out=None) -> dict:
    """Full CoverPrune (FST cost, capacity, SGS): kept [B,K] ascending, plus
    order [B,K], gains [B,K] and objective [B] when requested."""
    unbatched = feats.dim() == 2
    feats, pos, frame, B, N, D = _batched(feats, pos, frame)
    dt = _dtype(feats)
    params = params or Params()
    dev = feats.device
    out = dict(out or {})
    out.setdefault("kept", torch.empty(B, K, dtype=torch.int64, device=dev))
    if order:
        out.setdefault("order", torch.empty(B, K, dtype=torch.int64, device=dev))
    if gains:
        out.setdefault("gains", torch.empty(B, K, dtype=torch.float32, device=dev))
    if objective:
        out.setdefault("objective", torch.empty(B, dtype=torch.float64, device=dev))
    ws = _ws(ws, CP_OP_SELECT, B, N, D, K, dt, params, dev)
    p = params._c()
    _check(_lib().coverprune_select(_ptr(feats), dt, _ptr(pos), _ptr(frame), B, N, D, K,
                                    C.byref(p), _ptr(out["kept"]), _ptr(out.get("order")),
                                    _ptr(out.get("gains")), _ptr(out.get("objective")),
                                    _ptr(ws), ws.numel(), _stream()), "coverprune_select")
    if unbatched:
        out = {k: v[0] for k, v in out.items()}
    out["ws"] = ws
    return out


def coverprune_lite_select(feats, pos, frame, K: int, params: Params | None = None, *,
                           group_start=True, objective=True, ws=None, out=None) -> dict:
    """CoverPrune-Lite: kept [B,K] ascending, group_start [B,K+1], objective [B]."""
    unbatched = feats.dim() == 2
    feats, pos, frame, B, N, D = _batched(feats, pos, frame)
    dt = _dtype(feats)
    params = params or Params()
    dev = feats.device
    out = dict(out or {})
    out.setdefault("kept", torch.empty(B, K, dtype=torch.int64, device=dev))
    if group_start:
        out.setdefault("group_start", torch.empty(B, K + 1, dtype=torch.int32, device=dev))
    if objective:
        out.setdefault("objective", torch.empty(B, dtype=torch.float64, device=dev))
    ws = _ws(ws, CP_OP_LITE, B, N, D, K, dt, params, dev)
    p = params._c()
    _check(_lib().coverprune_lite_select(_ptr(feats), dt, _ptr(pos), _ptr(frame), B, N, D, K,
                                         C.byref(p), _ptr(out["kept"]),
                                         _ptr(out.get("group_start")),
                                         _ptr(out.get("objective")), _ptr(ws), ws.numel(),
                                         _stream()), "coverprune_lite_select")
    if unbatched:
        out = {k: v[0] for k, v in out.items()}
    out["ws"] = ws
    return out


def coverprune_knn(pos, k: int, *, diameter=True, ws=None):
    """(nbr int32 [B,N,k], diameter [B]): the k nearest other tokens of every
    token by (fp32 squared distance, index) and each scene's diameter."""
    unbatched = pos.dim() == 2
    if unbatched:
        pos = pos.unsqueeze(0)
    if not pos.is_cuda or not pos.is_contiguous() or pos.dtype != torch.float32:
        raise ValueError("pos must be a contiguous float32 CUDA tensor [B,N,3]")
    B, N, _ = pos.shape
    nbr = torch.empty(B, N, k, dtype=torch.int32, device=pos.device)
    dia = torch.empty(B, dtype=torch.float32, device=pos.device) if diameter else None
    if ws is None:
        ws = workspace(CP_OP_KNN, B, N, 8, 0, CP_BF16, None, pos.device)
    _check(_lib().coverprune_knn(_ptr(pos), B, N, k, _ptr(nbr), _ptr(dia), _ptr(ws), ws.numel(),
                                 _stream()), "coverprune_knn")
    if unbatched:
        return nbr[0], (dia[0] if dia is not None else None)
    return nbr, dia


def coverprune_knn_noalloc(pos, nbr, diameter=None) -> None:
    """coverprune_knn into caller-provided outputs, with no workspace: for
    hosts that cannot allocate device memory (the library uses a fixed
    internal scratch; at most 1024 scenes per call).  nbr is int32
    [B, N, k] (or [N, k]), diameter float32 [B] (or a 1-element tensor)."""
    if pos.dim() == 2:
        pos = pos.unsqueeze(0)
        nbr = nbr.unsqueeze(0)
    if not pos.is_cuda or not pos.is_contiguous() or pos.dtype != torch.float32:
        raise ValueError("pos must be a contiguous float32 CUDA tensor [B,N,3]")
    if nbr.dtype != torch.int32 or not nbr.is_contiguous():
        raise ValueError("nbr must be a contiguous int32 tensor [B,N,k]")
    B, N, _ = pos.shape
    k = nbr.shape[-1]
    _check(_lib().coverprune_knn_noalloc(_ptr(pos), B, N, k, _ptr(nbr), _ptr(diameter),
                                         _stream()), "coverprune_knn_noalloc")


def coverprune_gather(feats, pos, frame, kept, *, status=None, out=None):
    """(feats_out [B,K,D], pos_out [B,K,3], frame_out [B,K]) of the kept rows."""
    unbatched = feats.dim() == 2
    feats, pos, frame, B, N, D = _batched(feats, pos, frame)
    if unbatched:
        kept = kept.unsqueeze(0)
    if kept.dtype != torch.int64 or not kept.is_contiguous() or kept.shape[0] != B:
        raise ValueError("kept must be contiguous int64 [B, K]")
    K = kept.shape[1]
    dev = feats.device
    out = dict(out or {})
    fo = out.get("feats", torch.empty(B, K, D, dtype=feats.dtype, device=dev))
    po = out.get("pos", torch.empty(B, K, 3, dtype=torch.float32, device=dev))
    to = out.get("frame", torch.empty(B, K, dtype=torch.int32, device=dev))
    _check(_lib().coverprune_gather(_ptr(feats), _dtype(feats), _ptr(pos), _ptr(frame), B, N, D,
                                    _ptr(kept), K, _ptr(fo), _ptr(po), _ptr(to), _ptr(status),
                                    _stream()), "coverprune_gather")
    if unbatched:
        return fo[0], po[0], to[0]
    return fo, po, to


def coverprune_barrier_selftest(n_blocks: int, expected: int, timeout_ms: float, ws) -> int:
    """Launch the bounded grid-barrier self-test; returns the device status
    (CP_ETIMEOUT when expected > n_blocks)."""
    _check(_lib().coverprune_barrier_selftest(n_blocks, expected, timeout_ms, _ptr(ws),
                                              ws.numel(), _stream()),
           "coverprune_barrier_selftest")
    return coverprune_check(ws)


def coverprune_profile_enable(on: bool = True) -> None:
    _check(_lib().coverprune_profile_enable(1 if on else 0), "coverprune_profile_enable")


def coverprune_profile_read() -> dict:
    """{stage: (milliseconds, kernel launches)} since the previous read."""
    n = len(STAGES)
    ms = (C.c_double * n)()
    la = (C.c_int64 * n)()
    _check(_lib().coverprune_profile_read(ms, la, n), "coverprune_profile_read")
    return {name: (float(ms[i]), int(la[i])) for i, name in enumerate(STAGES)}


def coverprune_call_stats(ws) -> dict:
    """{"gain_evaluations", "rounds", "cost_bytes_read"} of the last
    coverprune_select on ws."""
    out = _CallStats()
    _check(_lib().coverprune_call_stats(_ptr(ws), _stream(), C.byref(out)),
           "coverprune_call_stats")
    return {"gain_evaluations": int(out.gain_evaluations), "rounds": int(out.rounds),
            "cost_bytes_read": int(out.cost_bytes_read)}


def coverprune_version() -> int:
    return int(_lib().coverprune_version())
