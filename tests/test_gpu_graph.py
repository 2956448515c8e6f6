"""The library's calls captured as a CUDA graph (as the benchmark times them):
a replay recomputes everything from the current contents of the input
buffers.  After new inputs are written into the same buffers, a replay's
packed cache and decode output equal a direct call on the new inputs bit for
bit, and differ from the first inputs' results."""
import numpy as np
import pytest
import torch

import parity
from paper_2608_21541_gb300 import certkv as ck
from paper_2608_21541_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def test_graph_replay_recomputes_from_current_inputs():
    wl = W.Workload("GR", B=1, L=2, Hq=8, H=2, n=9000, d=128, w=64, keep=(1, 10), kind="zipf")
    K, V, Q = W.draw(wl, seed=1, device="cuda")
    q = W.draw_decode_queries(wl, 0, seed=1, device="cuda")
    shape = ck.shape_of(K, Q)
    ws = ck.workspace(ck.certkv_workspace_bytes(shape), "cuda")
    dshape = ck.certkv_shape(wl.B, wl.L, wl.Hq, wl.H, 2, wl.d, 1)
    dws = ck.workspace(ck.certkv_decode_workspace_bytes(dshape), "cuda")
    packed = ck.Packed.empty(wl.B, wl.L, wl.H, wl.d, wl.B_live, "cuda", with_tail=True)
    out = torch.empty_like(q)

    def calls(st):
        ck.certkv_compress(K, V, Q, wl.B_live, out=packed, ws=ws, stream=st)
        ck.certkv_decode_attn(q, packed, hkv=wl.H, out=out, ws=dws, stream=st)

    def snapshot():
        torch.cuda.synchronize()
        res = parity.packed_np(packed)
        res["out"] = out.view(-1).view(torch.int16).cpu().numpy()
        return res

    calls(torch.cuda.current_stream())  # first use outside the capture
    first = snapshot()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        calls(torch.cuda.current_stream())
    g.replay()
    replay_first = snapshot()
    for k in first:
        np.testing.assert_array_equal(first[k], replay_first[k], err_msg=k)
    # new inputs in the same buffers
    K2, V2, Q2 = W.draw(wl, seed=2, device="cuda")
    K.copy_(K2), V.copy_(V2), Q.copy_(Q2)
    q.copy_(W.draw_decode_queries(wl, 0, seed=2, device="cuda"))
    g.replay()
    replay_second = snapshot()
    calls(torch.cuda.current_stream())
    direct_second = snapshot()
    for k in direct_second:
        np.testing.assert_array_equal(direct_second[k], replay_second[k], err_msg=k)
    assert not np.array_equal(first["positions"], replay_second["positions"])
    assert not np.array_equal(first["out"], replay_second["out"])
