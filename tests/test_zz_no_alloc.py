"""coverprune_knn_noalloc against coverprune_knn.

Callers that cannot allocate device memory (their host owns a fixed,
sealed memory pool, or they run as a plugin with no allocator) use the
workspace-free variant, whose scratch is a fixed array inside the library.
Its neighbour lists must be identical to those of the workspace entry point
(integers: bit-exact) and its diameters equal (same arithmetic), on two
calls in a row -- the second with different sizes and data, so that nothing
left in the shared scratch by the first call can leak into it.  This file is
collected last and also passes when run on its own in a fresh process.
"""
import ctypes as C

import numpy as np
import pytest
import torch

import paper_2608_13226_gb300 as cp

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2608_13226_gb300 import build
    build.build()
    cp.load()


def _positions(seed, B, N):
    rng = np.random.default_rng(seed)
    x = (rng.random((B, N, 3)) * np.array([8.0, 8.0, 3.0])).astype(np.float32)
    x[:, ::7] = x[:, 3:4]  # coincident points: exercises the index tie-break
    return torch.from_numpy(x).cuda()


# k = 8: the workspace entry point takes its grid kernel (lists in registers)
# and this one its brute-force kernel; k = 0: the scene diameter alone
@pytest.mark.parametrize("case", [(11, 3, 1500, 20), (12, 1, 777, 63), (13, 2, 1500, 8),
                                  (14, 2, 900, 0)])
def test_noalloc_matches_workspace_entry_point_twice(case):
    seed, B, N, k = case
    for call in range(2):  # two calls in a row; the second one changes sizes and data
        pos = _positions(seed + 100 * call, B + call, N - 13 * call)
        Bc, Nc = pos.shape[0], pos.shape[1]
        ref_nbr, ref_dia = cp.coverprune_knn(pos, k)
        nbr = torch.full((Bc, Nc, k), -1, dtype=torch.int32, device="cuda")
        dia = torch.full((Bc,), -1.0, dtype=torch.float32, device="cuda")
        cp.coverprune_knn_noalloc(pos, nbr, dia)
        torch.cuda.synchronize()
        assert torch.equal(nbr, ref_nbr), f"call {call}: neighbour lists differ"
        np.testing.assert_allclose(dia.cpu().numpy(), ref_dia.cpu().numpy(), rtol=1e-6, atol=0)


def test_noalloc_rejects_more_scenes_than_its_scratch():
    lib = cp.load()
    st = lib.coverprune_knn_noalloc(C.c_void_p(0x100000), 1025, 100, 4, C.c_void_p(0x100000),
                                    None, None)  # rejected before any launch
    assert st == cp.CP_EUNSUPPORTED
    assert "1024" in lib.coverprune_last_error().decode()
