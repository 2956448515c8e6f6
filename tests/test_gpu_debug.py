"""The bounds-checking build of the library (-DCERTKV_DEBUG: every ragged
index and offset is checked against its extent; a violation sets
CERTKV_STATUS_BOUNDS and skips the access, nothing traps) on small cases with
ragged sizes, several group sizes and head counts, cluster summaries and no
tail slot.  It runs in a child process (the library is chosen with
CERTKV_LIBRARY), must report no violation and leave every workspace guard
intact, and its outputs must equal the normal build's bit for bit: the checks
change no arithmetic."""
import multiprocessing as mp
import os
import sys

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

# (name, (B, L, Hq, H, n, w, keep, kind), params overrides)
CASES = [
    ("ragged", (2, 2, 8, 2, 3000, 20, (1, 10), "planted"), {}),
    ("mha_g1", (1, 1, 4, 4, 2500, 7, (1, 8), "lowrank"), {}),
    ("g8_rows512", (1, 2, 16, 2, 4100, 64, (1, 10), "zipf"), {}),
    ("heads32", (1, 1, 32, 32, 700, 4, (1, 5), "student_t"), {}),
    ("clusters", (1, 2, 8, 2, 2300, 16, (1, 8), "planted"), {"tail_clusters": 3}),
    ("no_tail_slot", (1, 1, 8, 2, 1800, 16, (1, 8), "zipf"), {"tail_slot": 0}),
    ("n2", (1, 2, 8, 4, 2, 1, (1, 1), "zipf"), {}),       # the smallest context
    ("n3_g16", (1, 1, 16, 1, 3, 2, (2, 3), "zipf"), {}),
    ("n64_h3", (2, 1, 12, 3, 64, 4, (1, 3), "planted"), {}),
]


def run_cases():
    """Every case through certkv_score, certkv_curves, certkv_compress and
    certkv_decode_attn on one guarded workspace; numpy outputs and the
    status word and guard count of each case."""
    import torch

    from paper_2608_21541_gb300 import certkv as ck
    from paper_2608_21541_gb300 import workloads as W
    out = {}
    for name, (B, L, Hq, H, n, w, keep, kind), over in CASES:
        wl = W.Workload(name, B=B, L=L, Hq=Hq, H=H, n=n, d=128, w=w, keep=keep, kind=kind)
        params = ck.certkv_default_params(**over)
        K, V, Q = W.draw(wl, device="cuda")
        shape = ck.shape_of(K, Q)
        ws = ck.workspace(ck.certkv_workspace_bytes(shape, params), "cuda")
        ck.certkv_workspace_guard_arm(ws, shape, params)
        a = ck.certkv_score(K, Q, params, ws=ws)
        st_score = ck.certkv_read_status(ws)
        perm, c = ck.certkv_curves(V, a, params, hq=Hq, w=w, ws=ws)
        st_curves = ck.certkv_read_status(ws)
        packed = ck.certkv_compress(K, V, Q, wl.B_live, params, ws=ws, with_tail=True)
        st_compress = ck.certkv_read_status(ws)
        guards = ck.certkv_workspace_guard_check(ws, shape, params)
        q = W.draw_decode_queries(wl, 0, device="cuda")
        dec = ck.certkv_decode_attn(q, packed, hkv=H)
        torch.cuda.synchronize()
        bits = lambda t: t.contiguous().cpu().view(torch.int16).numpy()
        out[name] = dict(
            status=(st_score, st_curves, st_compress), guards=guards,
            a=a.cpu().numpy(), perm=perm.cpu().numpy(), c=c.cpu().numpy(),
            counts=packed.real_counts.cpu().numpy(), offsets=packed.offsets.cpu().numpy(),
            positions=packed.positions.cpu().numpy(), pk=bits(packed.k), pv=bits(packed.v),
            dec=bits(dec))
    return out


def _child(q, lib):
    sys.path.insert(0, ROOT)
    os.environ["CERTKV_LIBRARY"] = lib
    try:
        q.put(("ok", run_cases()))
    except Exception as e:  # reported to the parent
        q.put(("error", repr(e)))


def test_debug_build_finds_nothing_and_matches_the_normal_build():
    from paper_2608_21541_gb300 import build as B
    from paper_2608_21541_gb300 import certkv as ck
    lib = B.build(debug=True)
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    p = ctx.Process(target=_child, args=(q, lib))
    p.start()
    kind, dbg = q.get(timeout=900)
    p.join(timeout=120)
    assert kind == "ok", dbg
    assert p.exitcode == 0
    ref = run_cases()  # the normal build, in this process
    for name, got in dbg.items():
        assert all(s & ck.STATUS_BOUNDS == 0 for s in got["status"]), (name, got["status"])
        assert got["status"] == ref[name]["status"], (name, got["status"], ref[name]["status"])
        assert got["guards"] == 0 and ref[name]["guards"] == 0, name
        for k in ("a", "perm", "c", "counts", "offsets", "positions", "pk", "pv", "dec"):
            assert np.array_equal(got[k], ref[name][k]), (name, k)
