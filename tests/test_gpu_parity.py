"""CUDA path versus the float64 oracle on seeded inputs, through the C ABI.

Sizes span several score tiles (64 keys), key splits (1024), sort tiles
(4096), dispersion chunks (128) and hull segments (1024), with ragged tails,
every supported group size pattern, more than one row block, the variants of
the parameters, and the extreme budgets."""
import numpy as np
import pytest
import torch

import oracle
import parity
from paper_2608_21541_gb300 import certkv as ck
from paper_2608_21541_gb300 import workloads as W

pytestmark = pytest.mark.gpu

DEV = "cuda"

CASES = {
    "small_ragged": W.Workload("S", B=2, L=2, Hq=8, H=2, n=3000, d=128, w=20, keep=(1, 10),
                               kind="planted"),
    "C1": W.WORKLOADS["C1"],
    "mha_g1": W.Workload("M", B=1, L=1, Hq=4, H=4, n=2500, d=128, w=7, keep=(1, 8),
                         kind="lowrank"),
    "gqa_g8_lowrank": W.Workload("G8", B=1, L=2, Hq=16, H=2, n=2049, d=128, w=9, keep=(1, 6),
                                 kind="lowrank"),
    "rows1024_student": W.Workload("T", B=1, L=1, Hq=32, H=2, n=1500, d=128, w=64, keep=(1, 5),
                                   kind="student_t"),
    "zipf_long": W.Workload("Z", B=1, L=1, Hq=8, H=2, n=9000, d=128, w=64, keep=(1, 10),
                            kind="zipf"),
    # R = G w = 512 and 768: the tcgen05 pass 2 in two and three 256-row groups
    "rows512_zipf": W.Workload("Z5", B=1, L=2, Hq=16, H=2, n=4100, d=128, w=64, keep=(1, 10),
                               kind="zipf"),
    "rows768_planted": W.Workload("P7", B=1, L=1, Hq=32, H=2, n=3333, d=128, w=48, keep=(1, 8),
                                  kind="planted"),
    # head counts that change the allocator's work split: one KV head (three
    # bisection steps per round), 16 and 32 heads (one step per round, one
    # warp per head at 32)
    "mqa_h1": W.Workload("Q1", B=1, L=1, Hq=8, H=1, n=2600, d=128, w=16, keep=(1, 10),
                         kind="zipf"),
    "heads16": W.Workload("H16", B=1, L=1, Hq=16, H=16, n=1200, d=128, w=8, keep=(1, 6),
                          kind="planted"),
    "heads32": W.Workload("H32", B=1, L=1, Hq=32, H=32, n=700, d=128, w=4, keep=(1, 5),
                          kind="student_t"),
}

_cache = {}


def run_case(name, wl=None, params=None, B_live=None, seed=0):
    key = (name, seed, None if params is None else tuple(getattr(params, f) for f, _ in
                                                          params._fields_), B_live)
    if key in _cache:
        return _cache[key]
    wl = wl or CASES[name]
    params = params or ck.certkv_default_params()
    B_live = B_live or wl.B_live
    K, V, Q = W.draw(wl, seed=seed, device=DEV)
    # one workspace for the three calls, with its guard words armed: no
    # kernel may write past the end of a region
    shape = ck.shape_of(K, Q)
    ws = ck.workspace(ck.certkv_workspace_bytes(shape, params), DEV)
    ck.certkv_workspace_guard_arm(ws, shape, params)
    a = ck.certkv_score(K, Q, params, ws=ws)
    packed = ck.certkv_compress(K, V, Q, B_live, params, ws=ws, with_tail=True)
    scored = ck.certkv_compress_scored(K, V, a, B_live, params, hq=wl.Hq, w=wl.w, ws=ws,
                                       with_tail=True)
    torch.cuda.synchronize()
    guards = ck.certkv_workspace_guard_check(ws, shape, params)
    status = ck.certkv_read_status(ws)
    host = dict(K=parity.bits(K), V=parity.bits(V), Q=parity.bits(Q),
                a=a.cpu().numpy())
    kw = dict(B=wl.B, L=wl.L, Hq=wl.Hq, H=wl.H, n=wl.n, d=wl.d, w=wl.w, B_live=B_live,
              scale=params.scale, pool=params.pool_kernel, protect=params.protect_window,
              alpha_num=params.alpha_num, alpha_den=params.alpha_den, T=params.bisect_steps,
              statistic=params.statistic, tail_slot=params.tail_slot,
              allocator=params.allocator)
    ref_e2e = oracle.compress(host["K"], host["V"], host["Q"], **kw)
    ref_cond = oracle.compress(host["K"], host["V"], None, a_in=host["a"], **kw)
    res = dict(wl=wl, params=params, B_live=B_live, K=K, V=V, Q=Q, a=a, packed=packed,
               scored=scored, host=host, ref_e2e=ref_e2e, ref_cond=ref_cond, guards=guards,
               status=status)
    _cache[key] = res
    return res


@pytest.mark.parametrize("name", sorted(CASES))
def test_workspace_guards_intact(name):
    """After certkv_score, certkv_compress and certkv_compress_scored on one
    workspace, every region's guard words still hold their pattern."""
    r = run_case(name)
    assert r["guards"] == 0, f"{r['guards']} workspace guard words overwritten"
    assert r["status"] == 0, r["status"]


@pytest.mark.parametrize("name", sorted(CASES))
def test_scores_match_oracle(name):
    r = run_case(name)
    parity.check_scores(r["host"]["a"], r["ref_e2e"]["a"])


@pytest.mark.parametrize("name", sorted(CASES))
def test_order_and_curves_conditioned(name):
    r = run_case(name)
    wl = r["wl"]
    perm, c = ck.certkv_curves(r["V"], r["a"], hq=wl.Hq, w=wl.w)
    perm, c = perm.cpu().numpy(), c.cpu().numpy()
    ref = r["ref_cond"]
    np.testing.assert_array_equal(perm, ref["perm"])
    rel = np.abs(c - ref["c"]) / np.maximum(np.abs(ref["c"]).max(axis=1, keepdims=True), 1e-300)
    assert rel.max() < 1e-8, rel.max()


@pytest.mark.parametrize("name", sorted(CASES))
def test_compress_conditioned_bit_exact(name):
    r = run_case(name)
    got = parity.packed_np(r["scored"])
    parity.check_conditioned(got, r["ref_cond"], r["wl"].units)


@pytest.mark.parametrize("name", sorted(CASES))
def test_compress_pass_equals_scored_path(name):
    """certkv_compress = certkv_score followed by certkv_compress_scored."""
    r = run_case(name)
    a1, a2 = parity.packed_np(r["packed"]), parity.packed_np(r["scored"])
    for k in ("counts", "offsets", "positions", "pk", "pv"):
        np.testing.assert_array_equal(a1[k], a2[k], err_msg=k)


@pytest.mark.parametrize("name", sorted(CASES))
def test_compress_pass_conditioned(name):
    """certkv_compress itself against the oracle conditioned on the same
    scores: budgets, positions and real slots bit-exact, tail mass and
    centroids within 1e-4."""
    r = run_case(name)
    parity.check_conditioned(parity.packed_np(r["packed"]), r["ref_cond"], r["wl"].units)


@pytest.mark.parametrize("name", sorted(CASES))
def test_compress_end_to_end(name):
    r = run_case(name)
    got = parity.packed_np(r["packed"])
    parity.check_end_to_end(got, r["ref_e2e"], r["host"]["a"], r["wl"].H)
    assert got["counts"].reshape(-1, r["wl"].H).sum(1).tolist() == \
        [r["B_live"] - r["wl"].H] * (r["wl"].B * r["wl"].L)


@pytest.mark.parametrize("name", sorted(CASES))
def test_decode_matches_oracle(name):
    r = run_case(name)
    wl = r["wl"]
    got = parity.packed_np(r["packed"])
    for step in (0, 1):
        q = W.draw_decode_queries(wl, step, device=DEV)
        out = ck.certkv_decode_attn(q, r["packed"], hkv=wl.H)
        ref = oracle.decode(parity.bits(q), got["pk"], got["pv"], got["offsets"], got["counts"],
                            B=wl.B, L=wl.L, Hq=wl.Hq, H=wl.H, d=wl.d)
        parity.check_decode(out, ref)


# ---------------------------------------------------------------- variants --

VARIANTS = {
    "uncentered": dict(statistic=1),
    "tail_mass": dict(statistic=2),
    "no_tail_slot": dict(tail_slot=0),
    "no_bisection": dict(bisect_steps=0),
    "alpha0": dict(alpha_num=0, alpha_den=1),
    "alpha04": dict(alpha_num=2, alpha_den=5),
    "no_pool_no_protect": dict(pool_kernel=1, protect_window=0),
    "pool7_scale": dict(pool_kernel=7, scale=0.05),
    "allocator_uniform": dict(allocator=1),
    "allocator_greedy": dict(allocator=2),
}


@pytest.mark.parametrize("var", sorted(VARIANTS))
def test_parameter_variants_conditioned(var):
    params = ck.certkv_default_params(**VARIANTS[var])
    r = run_case("small_ragged", params=params)
    parity.check_scores(r["host"]["a"], r["ref_e2e"]["a"])
    got = parity.packed_np(r["scored"])
    parity.check_conditioned(got, r["ref_cond"], r["wl"].units, tail_slot=params.tail_slot)
    q = W.draw_decode_queries(r["wl"], 0, device=DEV)
    packed = r["scored"]
    out = ck.certkv_decode_attn(q, packed, hkv=r["wl"].H)
    ref = oracle.decode(parity.bits(q), got["pk"], got["pv"], got["offsets"], got["counts"],
                        B=r["wl"].B, L=r["wl"].L, Hq=r["wl"].Hq, H=r["wl"].H, d=128,
                        tail_slot=params.tail_slot)
    parity.check_decode(out, ref)


@pytest.mark.parametrize("which", ["min", "max", "tiny_n"])
def test_extreme_budgets(which):
    wl = CASES["small_ragged"]
    if which == "tiny_n":
        wl = wl.with_(n=34, w=32, L=1)
        B_live = 3 * wl.H
    elif which == "min":
        B_live = 2 * wl.H            # one real token per head
    else:
        B_live = wl.H * wl.n         # every head keeps n - 1 real tokens
    r = run_case(f"extreme_{which}", wl=wl, B_live=B_live)
    got = parity.packed_np(r["scored"])
    parity.check_conditioned(got, r["ref_cond"], wl.units)
    if which == "max":
        assert (got["counts"] == wl.n - 1).all()
    if which == "min":
        assert (got["counts"] == 1).all()


def test_deterministic():
    wl = CASES["small_ragged"]
    K, V, Q = W.draw(wl, device=DEV)
    p1 = parity.packed_np(ck.certkv_compress(K, V, Q, wl.B_live, with_tail=True))
    p2 = parity.packed_np(ck.certkv_compress(K, V, Q, wl.B_live, with_tail=True))
    for k in p1:
        np.testing.assert_array_equal(p1[k], p2[k], err_msg=k)


@pytest.mark.parametrize("where", ["K_nan", "V_nan", "V_inf", "Q_inf"])
def test_status_word_nonfinite_inputs(where):
    """A NaN or an infinity in K, V or the observation queries raises
    CERTKV_STATUS_NONFINITE (the call returns normally), and the next call
    with finite inputs on the same workspace reports a clean status again."""
    wl = CASES["small_ragged"]
    K, V, Q = W.draw(wl, device=DEV)
    shape = ck.shape_of(K, Q)
    ws = ck.workspace(ck.certkv_workspace_bytes(shape), K.device)
    bad = {"K": K.clone(), "V": V.clone(), "Q": Q.clone()}
    name, kind = where.split("_")
    bad[name].view(-1)[1234] = float("nan") if kind == "nan" else float("inf")
    ck.certkv_compress(bad["K"], bad["V"], bad["Q"], wl.B_live, ws=ws)
    assert ck.certkv_read_status(ws) & ck.STATUS_NONFINITE
    ck.certkv_compress(K, V, Q, wl.B_live, ws=ws)
    assert ck.certkv_read_status(ws) == 0


def test_status_word():
    wl = CASES["small_ragged"]
    K, V, Q = W.draw(wl, device=DEV)
    shape = ck.shape_of(K, Q)
    ws = ck.workspace(ck.certkv_workspace_bytes(shape), K.device)
    ck.certkv_compress(K, V, Q, wl.B_live, ws=ws)
    assert ck.certkv_read_status(ws) == 0
    K2 = K.clone()
    K2[0, 0, 0, 5, 3] = float("nan")
    ck.certkv_compress(K2, V, Q, wl.B_live, ws=ws)
    assert ck.certkv_read_status(ws) & ck.STATUS_NONFINITE
