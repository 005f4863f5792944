"""Failure detection without a GPU fault: every device-side wait of the
library is bounded.  The self-test launches co-resident blocks on a grid
barrier that expects more arrivals than there are blocks -- a flag nobody
sets -- and the kernel must give up after the time limit, record
CP_ETIMEOUT in the workspace status word and return, leaving the context
usable."""
import time

import pytest
import torch

import paper_2608_13226_gb300 as cp

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2608_13226_gb300 import build
    build.build()
    cp.load()


def test_barrier_times_out_and_context_survives():
    ws = torch.empty(256, dtype=torch.uint8, device="cuda")
    t0 = time.time()
    st = cp.coverprune_barrier_selftest(4, 5, 50.0, ws)  # 4 blocks, 5 expected
    dt = time.time() - t0
    assert st == cp.CP_ETIMEOUT
    assert dt < 5.0
    # the context still works: a passing barrier and a real call
    assert cp.coverprune_barrier_selftest(4, 4, 50.0, ws) == cp.CP_OK
    f = torch.randn(64, 16, device="cuda").to(torch.bfloat16)
    pos = torch.rand(64, 3, device="cuda")
    fr = torch.zeros(64, dtype=torch.int32, device="cuda")
    r = cp.coverprune_select(f, pos, fr, 8)
    assert cp.coverprune_check(r["ws"]) == cp.CP_OK
    assert r["kept"].shape == (8,)


def test_select_reports_ok_status():
    f = torch.randn(300, 64, device="cuda").to(torch.bfloat16)
    pos = torch.rand(300, 3, device="cuda")
    fr = torch.arange(300, dtype=torch.int32, device="cuda") // 30
    for g in (0, 12):
        r = cp.coverprune_select(f, pos, fr, 30, cp.Params(g=g))
        assert cp.coverprune_check(r["ws"]) == cp.CP_OK
    lt = cp.coverprune_lite_select(f, pos, fr, 30)
    assert cp.coverprune_check(lt["ws"]) == cp.CP_OK
