"""The bounded waits: a wait on an mbarrier that nothing arrives on (no copy
and no MMA outstanding) gives up after its poll limit, reports
CERTKV_STATUS_TIMEOUT and leaves the context usable (a compression pass
right after it still matches the oracle's budgets)."""
import time

import pytest
import torch

import oracle
from paper_2608_21541_gb300 import certkv as ck
from paper_2608_21541_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def test_bounded_wait_gives_up_and_the_context_stays_usable():
    lib = ck.load_library()
    t0 = time.perf_counter()
    rc = lib.certkv_selftest_bounded_wait(None)
    took = time.perf_counter() - t0
    assert rc == ck.STATUS_TIMEOUT, rc
    assert took < 60.0, took
    wl = W.Workload("A", B=1, L=1, Hq=8, H=2, n=1500, d=128, w=16, keep=(1, 8), kind="planted")
    K, V, Q = W.draw(wl, device="cuda")
    packed = ck.certkv_compress(K, V, Q, wl.B_live)
    torch.cuda.synchronize()
    ref = oracle.compress(W.bf16_bits(K), W.bf16_bits(V), W.bf16_bits(Q), B=1, L=1, Hq=wl.Hq,
                          H=wl.H, n=wl.n, d=wl.d, w=wl.w, B_live=wl.B_live)
    assert (packed.real_counts.cpu().numpy() == ref["counts"]).all()
