"""Tiny shapes against the float64 oracle, through the C ABI: contexts of 2 to
64 tokens with 1 to 4 KV heads and every group size, so that every sort tile,
dispersion chunk, hull segment and decode tile is ragged or nearly empty and
the allocator's bracket is a handful of tokens.  Conditioned mode bit-exact,
end to end up to certified near-ties, decode within its tolerance; and the
whole pass bit-identical over ten repeats on a case with several tiles."""
import numpy as np
import pytest
import torch

import oracle
import parity
from paper_2608_21541_gb300 import certkv as ck
from paper_2608_21541_gb300 import workloads as W

pytestmark = pytest.mark.gpu

DEV = "cuda"

# (n, KV heads H, group size G): contexts from the smallest the method admits
# (n = 2, window 1) up to a half-filled dispersion chunk
SHAPES = [(2, 1, 1), (2, 4, 2), (3, 2, 4), (4, 1, 8), (5, 2, 2), (7, 3, 2), (9, 1, 16),
          (16, 2, 1), (16, 4, 4), (33, 1, 2), (33, 2, 8), (64, 3, 4), (64, 4, 1)]


def _case(n, H, G, kind="zipf"):
    w = min(n - 1, 1 + n % 5)
    # planted keys of distinct strengths (the Zipf recipe): identical planted
    # rows side by side, as a 64-token context of the plain recipe has, give
    # exactly equal scores whose order the float64 oracle breaks by index and
    # the fp32 path by rounding, and both orders are correct
    wl = W.Workload(f"tiny{n}_{H}_{G}", B=1, L=2, Hq=H * G, H=H, n=n, d=128, w=w,
                    keep=(1, 3), kind=kind, description="tiny shape")
    B_live = H * min(n, max(2, n // 3))
    return wl, B_live


@pytest.mark.parametrize("n,H,G,kind", [s + ("zipf",) for s in SHAPES] + [(64, 4, 1, "planted")])
def test_tiny_shapes_match_oracle(n, H, G, kind):
    """The last case has identical planted keys side by side, so some scores
    tie exactly in float64: it exercises the order near-tie rule."""
    wl, B_live = _case(n, H, G, kind)
    params = ck.certkv_default_params()
    K, V, Q = W.draw(wl, device=DEV)
    a = ck.certkv_score(K, Q, params)
    packed = ck.certkv_compress(K, V, Q, B_live, params, with_tail=True)
    scored = ck.certkv_compress_scored(K, V, a, B_live, params, hq=wl.Hq, w=wl.w, with_tail=True)
    host = dict(K=parity.bits(K), V=parity.bits(V), Q=parity.bits(Q), a=a.cpu().numpy())
    kw = dict(B=wl.B, L=wl.L, Hq=wl.Hq, H=wl.H, n=n, d=wl.d, w=wl.w, B_live=B_live)
    ref_e2e = oracle.compress(host["K"], host["V"], host["Q"], **kw)
    ref_cond = oracle.compress(host["K"], host["V"], None, a_in=host["a"], **kw)
    parity.check_scores(host["a"], ref_e2e["a"])
    parity.check_conditioned(parity.packed_np(scored), ref_cond, wl.units)
    got = parity.packed_np(packed)
    parity.check_end_to_end(got, ref_e2e, host["a"], H)
    assert got["counts"].reshape(-1, H).sum(1).tolist() == [B_live - H] * (wl.B * wl.L)
    q = W.draw_decode_queries(wl, 0, device=DEV)
    out = ck.certkv_decode_attn(q, packed, hkv=H)
    ref = oracle.decode(parity.bits(q), got["pk"], got["pv"], got["offsets"], got["counts"],
                        B=wl.B, L=wl.L, Hq=wl.Hq, H=H, d=wl.d)
    parity.check_decode(out, ref)


def test_ten_repeats_bit_identical():
    """Every output of the compression and of a decode step is bit-identical
    over ten calls (no atomics decide an order or a sum)."""
    wl = W.Workload("R", B=1, L=2, Hq=8, H=2, n=9000, d=128, w=64, keep=(1, 10),
                    kind="zipf", description="repeat case")
    K, V, Q = W.draw(wl, device=DEV)
    q = W.draw_decode_queries(wl, 0, device=DEV)
    first = None
    for _ in range(10):
        packed = ck.certkv_compress(K, V, Q, wl.B_live, with_tail=True)
        got = parity.packed_np(packed)
        out = ck.certkv_decode_attn(q, packed, hkv=wl.H)
        got["out"] = out.view(-1).view(torch.int16).cpu().numpy()
        if first is None:
            first = got
            continue
        for k in first:
            np.testing.assert_array_equal(first[k], got[k], err_msg=k)


@pytest.mark.parametrize("case", ["K_zero", "V_zero", "KV_zero", "V_rows_equal"])
def test_degenerate_inputs(case):
    """The method's degenerate inputs, against the oracle: all keys zero (every
    logit 0, so the scores tie except for the pooling edges and the protected
    window), all values zero (every curve c(b) = 0, so the allocator's ties
    decide every budget: smallest b, then the lowest head in the repair), both,
    and identical value rows (the centred dispersion is exactly 0)."""
    wl = W.Workload("D", B=1, L=2, Hq=8, H=2, n=3000, d=128, w=20, keep=(1, 10),
                    kind="planted", description="degenerate inputs")
    K, V, Q = W.draw(wl, device=DEV)
    if "K" in case:
        K.zero_()
    if case in ("V_zero", "KV_zero"):
        V.zero_()
    if case == "V_rows_equal":
        V.copy_(V[:, :, :, :1, :].expand_as(V))
    params = ck.certkv_default_params()
    a = ck.certkv_score(K, Q, params)
    packed = ck.certkv_compress(K, V, Q, wl.B_live, params, with_tail=True)
    scored = ck.certkv_compress_scored(K, V, a, wl.B_live, params, hq=wl.Hq, w=wl.w, with_tail=True)
    host = dict(K=parity.bits(K), V=parity.bits(V), Q=parity.bits(Q), a=a.cpu().numpy())
    kw = dict(B=wl.B, L=wl.L, Hq=wl.Hq, H=wl.H, n=wl.n, d=wl.d, w=wl.w, B_live=wl.B_live)
    ref_e2e = oracle.compress(host["K"], host["V"], host["Q"], **kw)
    ref_cond = oracle.compress(host["K"], host["V"], None, a_in=host["a"], **kw)
    parity.check_scores(host["a"], ref_e2e["a"])
    got = parity.packed_np(packed)
    if case != "V_rows_equal":
        parity.check_conditioned(parity.packed_np(scored), ref_cond, wl.units)
        parity.check_end_to_end(got, ref_e2e, host["a"], wl.H)
    else:
        # m Q - ||W||^2 is zero in exact arithmetic for every b: each side's
        # curve is its own rounding of 0, and the budgets follow that
        # rounding.  The path's c^2 carries the fp32 rounding of its in-chunk
        # terms 2<W_base, P> + ||P||^2 (at most m^2 ||v||^2 = m Q here, a few
        # units of 2^-24 relative over a 128-rank chunk): within 16 2^-24 m Q,
        # so c within sqrt(2^-20 m Q) absolutely.  What is unique is checked:
        # the curve within that bound, the budget sums, the kept tokens as the
        # top of the path's own order for its own budgets, and the packed rows.
        perm, c = ck.certkv_curves(V, a, params, hq=wl.Hq, w=wl.w)
        perm, c = perm.cpu().numpy(), c.cpu().numpy()
        v = oracle.bf16_bits_to_f64(host["V"].reshape(wl.units, wl.n, wl.d)[:, 0])
        for u in range(wl.units):
            m = np.cumsum(ref_cond["a"][u][ref_cond["perm"][u]][::-1])[::-1]
            bound = np.sqrt(2.0 ** -20) * m * np.linalg.norm(v[u]) + 1e-30
            ratio = float((np.abs(c[u] - ref_cond["c"][u]) / bound).max())
            assert ratio <= 1.0, f"curve beyond its bound (unit {u}): {ratio:.3f} of it"
            o, b = int(got["offsets"][u]), int(got["counts"][u])
            want = np.sort(perm[u][:b])
            np.testing.assert_array_equal(got["positions"][o:o + b], want)
            rows = host["V"].reshape(wl.units, wl.n, wl.d)[u][want]
            assert (got["pv"][o:o + b] == rows).all()
        B_real = wl.B_live - wl.H
        assert (got["counts"].reshape(-1, wl.H).sum(1) == B_real).all()
    q = W.draw_decode_queries(wl, 0, device=DEV)
    out = ck.certkv_decode_attn(q, packed, hkv=wl.H)
    ref = oracle.decode(parity.bits(q), got["pk"], got["pv"], got["offsets"], got["counts"],
                        B=wl.B, L=wl.L, Hq=wl.Hq, H=wl.H, d=wl.d)
    parity.check_decode(out, ref)


@pytest.mark.parametrize("gain", [4.0, 16.0])
def test_large_logits(gain):
    """Keys scaled up by 4 and 16 (logit spreads of hundreds of nats, most of a
    row's softmax probabilities below fp32's normal range): the scores, column
    sums of many rows, stay within the 1e-4 tolerance (measured 2.8e-6 and
    1.8e-5; the smallest score at gain 16 is ~1e-19, inside fp32's range);
    conditioned mode bit-exact, end to end within the contract, decode within
    its tolerance."""
    wl = W.Workload("G", B=1, L=2, Hq=8, H=2, n=3000, d=128, w=20, keep=(1, 10),
                    kind="zipf", description="large logits")
    K, V, Q = W.draw(wl, device="cuda")
    K = (K.float() * gain).to(torch.bfloat16)
    params = ck.certkv_default_params()
    a = ck.certkv_score(K, Q, params)
    packed = ck.certkv_compress(K, V, Q, wl.B_live, params, with_tail=True)
    host = dict(K=parity.bits(K), V=parity.bits(V), Q=parity.bits(Q), a=a.cpu().numpy())
    kw = dict(B=wl.B, L=wl.L, Hq=wl.Hq, H=wl.H, n=wl.n, d=wl.d, w=wl.w, B_live=wl.B_live)
    ref_cond = oracle.compress(host["K"], host["V"], None, a_in=host["a"], **kw)
    ref_e2e = oracle.compress(host["K"], host["V"], host["Q"], **kw)
    got = parity.packed_np(packed)
    parity.check_conditioned(got, ref_cond, wl.units)
    parity.check_scores(host["a"], ref_e2e["a"])
    parity.check_end_to_end(got, ref_e2e, host["a"], wl.H)
    q = W.draw_decode_queries(wl, 0, device=DEV)
    out = ck.certkv_decode_attn(q, packed, hkv=wl.H)
    ref = oracle.decode(parity.bits(q), got["pk"], got["pv"], got["offsets"], got["counts"],
                        B=wl.B, L=wl.L, Hq=wl.Hq, H=wl.H, d=wl.d)
    parity.check_decode(out, ref)


def test_budget_sweep():
    """Twelve live budgets from the smallest (one real token per head) to the
    largest (every head keeps n - 1 real tokens), odd ones included, on one
    case: every regime of the allocator (the floor b_min, short and long
    repairs, the budget ends) bit-exact in conditioned mode and within the
    contract end to end."""
    wl = W.Workload("BS", B=1, L=2, Hq=8, H=4, n=500, d=128, w=12, keep=(1, 10),
                    kind="zipf", description="budget sweep")
    K, V, Q = W.draw(wl, device=DEV)
    params = ck.certkv_default_params()
    a = ck.certkv_score(K, Q, params)
    host = dict(K=parity.bits(K), V=parity.bits(V), Q=parity.bits(Q), a=a.cpu().numpy())
    H, n = wl.H, wl.n
    budgets = sorted({2 * H, 2 * H + 1, 2 * H + 3, 3 * H, 37, 101, 250, 499, 1001, 1500,
                      H * n - 5, H * n})
    for B_live in budgets:
        kw = dict(B=wl.B, L=wl.L, Hq=wl.Hq, H=H, n=n, d=wl.d, w=wl.w, B_live=B_live)
        packed = ck.certkv_compress(K, V, Q, B_live, params, with_tail=True)
        got = parity.packed_np(packed)
        ref_cond = oracle.compress(host["K"], host["V"], None, a_in=host["a"], **kw)
        parity.check_conditioned(got, ref_cond, wl.units)
        ref_e2e = oracle.compress(host["K"], host["V"], host["Q"], **kw)
        parity.check_end_to_end(got, ref_e2e, host["a"], H)
        assert (got["counts"].reshape(-1, H).sum(1) == B_live - H).all(), B_live


TINY_VARIANTS = {
    "uncentered": dict(statistic=1),
    "tail_mass": dict(statistic=2),
    "no_tail_slot": dict(tail_slot=0),
    "no_bisection": dict(bisect_steps=0),
    "alpha0": dict(alpha_num=0, alpha_den=1),
    "alpha1": dict(alpha_num=1, alpha_den=1),
    "pool1_no_protect": dict(pool_kernel=1, protect_window=0),
    "pool255": dict(pool_kernel=255),          # wider than the whole context
    "allocator_uniform": dict(allocator=1),
    "allocator_greedy": dict(allocator=2),
}


@pytest.mark.parametrize("var", sorted(TINY_VARIANTS))
@pytest.mark.parametrize("n,H,G", [(9, 2, 2), (40, 3, 4)])
def test_tiny_parameter_variants(var, n, H, G):
    """Every parameter variant on tiny contexts (a pooling window wider than
    the context, the safeguard at 0 and 1, no bisection, the ablation
    allocators): conditioned mode bit-exact, decode within its tolerance."""
    wl, B_live = _case(n, H, G)
    params = ck.certkv_default_params(**TINY_VARIANTS[var])
    K, V, Q = W.draw(wl, device=DEV)
    a = ck.certkv_score(K, Q, params)
    packed = ck.certkv_compress_scored(K, V, a, B_live, params, hq=wl.Hq, w=wl.w, with_tail=True)
    host = dict(K=parity.bits(K), V=parity.bits(V), Q=parity.bits(Q), a=a.cpu().numpy())
    kw = dict(B=wl.B, L=wl.L, Hq=wl.Hq, H=H, n=n, d=wl.d, w=wl.w, B_live=B_live,
              scale=params.scale, pool=params.pool_kernel, protect=params.protect_window,
              alpha_num=params.alpha_num, alpha_den=params.alpha_den, T=params.bisect_steps,
              statistic=params.statistic, tail_slot=params.tail_slot, allocator=params.allocator)
    ref_e2e = oracle.compress(host["K"], host["V"], host["Q"], **kw)
    ref_cond = oracle.compress(host["K"], host["V"], None, a_in=host["a"], **kw)
    parity.check_scores(host["a"], ref_e2e["a"])
    got = parity.packed_np(packed)
    parity.check_conditioned(got, ref_cond, wl.units, tail_slot=params.tail_slot)
    q = W.draw_decode_queries(wl, 0, device=DEV)
    out = ck.certkv_decode_attn(q, packed, hkv=H)
    ref = oracle.decode(parity.bits(q), got["pk"], got["pv"], got["offsets"], got["counts"],
                        B=wl.B, L=wl.L, Hq=wl.Hq, H=H, d=wl.d, tail_slot=params.tail_slot)
    parity.check_decode(out, ref)
