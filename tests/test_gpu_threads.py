"""Two host threads using the library at the same time, each with its own
stream, workspace and packed cache (ctypes releases the interpreter lock
during each call, so the calls really overlap): every output of the
compression and of a decode step equals a call made alone, bit for bit, over
several rounds.  The library's process-wide state (kernel attributes set
once, cached occupancy figures) is written with the same values by whichever
call comes first."""
import threading

import numpy as np
import pytest
import torch

import parity
from paper_2608_21541_gb300 import certkv as ck
from paper_2608_21541_gb300 import workloads as W

pytestmark = pytest.mark.gpu

CASES = [W.Workload("T1", B=1, L=2, Hq=8, H=2, n=9000, d=128, w=64, keep=(1, 10), kind="zipf"),
         W.Workload("T2", B=2, L=1, Hq=16, H=2, n=5000, d=128, w=32, keep=(1, 8), kind="planted")]


def _run(wl, K, V, Q, q, stream, ws, dws, packed, out):
    with torch.cuda.stream(stream):
        ck.certkv_compress(K, V, Q, wl.B_live, out=packed, ws=ws, stream=stream)
        ck.certkv_decode_attn(q, packed, hkv=wl.H, out=out, ws=dws, stream=stream)
    stream.synchronize()
    res = parity.packed_np(packed)
    res["out"] = out.view(-1).view(torch.int16).cpu().numpy()
    return res


def test_two_threads_match_single_calls():
    setups = []
    for wl in CASES:
        K, V, Q = W.draw(wl, device="cuda")
        q = W.draw_decode_queries(wl, 0, device="cuda")
        shape = ck.shape_of(K, Q)
        ws = ck.workspace(ck.certkv_workspace_bytes(shape), "cuda")
        dshape = ck.certkv_shape(wl.B, wl.L, wl.Hq, wl.H, 2, wl.d, 1)
        dws = ck.workspace(ck.certkv_decode_workspace_bytes(dshape), "cuda")
        packed = ck.Packed.empty(wl.B, wl.L, wl.H, wl.d, wl.B_live, "cuda", with_tail=True)
        out = torch.empty_like(q)
        setups.append((wl, K, V, Q, q, torch.cuda.Stream(), ws, dws, packed, out))
    alone = [_run(*s) for s in setups]
    errors = []

    def worker(i):
        try:
            for _ in range(5):
                got = _run(*setups[i])
                for k in alone[i]:
                    if not np.array_equal(alone[i][k], got[k]):
                        errors.append(f"thread {i}: {k} differs")
                        return
        except Exception as e:  # reported by the main thread
            errors.append(f"thread {i}: {e!r}")

    threads = [threading.Thread(target=worker, args=(i,)) for i in range(len(setups))]
    for t in threads:
        t.start()
    for t in threads:
        t.join(timeout=300)
    assert not any(t.is_alive() for t in threads), "a thread did not finish"
    assert not errors, errors
