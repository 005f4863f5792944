"""GB300-native (sm_103a) hot path of CoverPrune, coverage-driven token
pruning for 3D VLMs via optimal transport.

The compute lives in ``libcoverprune.so`` (hand-written CUDA, C ABI in
``include/coverprune.h``); this package holds its build script, a thin ctypes
binding with the same entry-point names, and the seeded synthetic scene
generator used by the tests and the benchmark.
"""
from .binding import (CP_BF16, CP_EINVAL, CP_ETIMEOUT, CP_EUNSUPPORTED, CP_EWORKSPACE, CP_F32,
                      CP_OK, CP_OP_COST, CP_OP_KNN, CP_OP_LITE, CP_OP_SELECT, EXPORTS, CoverPruneError,
                      Params, coverprune_barrier_selftest, coverprune_budget, coverprune_call_stats, coverprune_check,
                      coverprune_cost, coverprune_gather, coverprune_knn, coverprune_knn_noalloc,
                      coverprune_lite_select,
                      coverprune_select, coverprune_version, coverprune_workspace_size,
                      library_path, load, status_string, workspace, coverprune_profile_enable,
                      coverprune_profile_read, STAGES)

__all__ = [n for n in dir() if not n.startswith("_")]
