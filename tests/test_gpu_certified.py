"""Clustered tail summaries and the certified decode (appendix: deterministic
output-error bound for clustered tail summaries) on the GPU against the
float64 oracle, in conditioned mode (the oracle starts from the GPU scores), and
the bound checked against exact attention over every original token."""
import numpy as np
import pytest
import torch

import oracle
import parity
from paper_2608_21541_gb300 import certkv as ck
from paper_2608_21541_gb300 import workloads as W

pytestmark = pytest.mark.gpu

WL = W.Workload("S", B=2, L=2, Hq=8, H=2, n=3000, d=128, w=20, keep=(1, 10), kind="planted")
# a 40-token context with 8 query heads per KV head: tails of about 30 tokens
# in up to 8 clusters, and as few as one real token per head
WLS = {"small": WL,
       "tiny40": W.Workload("T", B=1, L=2, Hq=16, H=2, n=40, d=128, w=3, keep=(1, 4),
                            kind="zipf")}
RADIUS_RTOL = 2e-5   # GPU radii are rounded up by 1e-5 relative; fp32 sums within 1e-5


def _run(m, tail_slot, WL=WL):
    K, V, Q = W.draw(WL, device="cuda")
    params = ck.certkv_default_params(tail_clusters=m, tail_slot=tail_slot)
    a = ck.certkv_score(K, Q, params)
    packed = ck.certkv_compress_scored(K, V, a, WL.B_live, params, hq=WL.Hq, w=WL.w)
    torch.cuda.synchronize()
    host = dict(K=parity.bits(K), V=parity.bits(V), a=a.cpu().numpy())
    ref = oracle.compress(host["K"], host["V"], None, a_in=host["a"], B=WL.B, L=WL.L, Hq=WL.Hq,
                          H=WL.H, n=WL.n, d=WL.d, w=WL.w, B_live=WL.B_live,
                          tail_slot=tail_slot, clusters=m)
    return K, V, Q, params, packed, ref, host


@pytest.mark.parametrize("wl", sorted(WLS))
@pytest.mark.parametrize("m,tail_slot", [(3, 1), (4, 0), (1, 1)])
def test_cluster_summaries_match_oracle(m, tail_slot, wl):
    K, V, Q, params, packed, ref, host = _run(m, tail_slot, WLS[wl])
    got = parity.packed_np(packed)
    assert (got["counts"] == ref["counts"]).all()
    assert (got["offsets"] == ref["offsets"]).all()
    assert (got["positions"] == ref["positions"]).all()
    meta = packed.cluster_meta.cpu().numpy().astype(np.float64)
    assert (meta[..., 0] == ref["cl_meta"][:, :m, 0]).all()
    for col in (1, 2):  # radii: valid upper bounds, tight to RADIUS_RTOL
        g, r = meta[..., col], ref["cl_meta"][:, :m, col]
        assert (g >= r * (1 - 1e-7)).all() and (g <= r * (1 + RADIUS_RTOL) + 1e-30).all()
    vm, rvm = packed.kept_vmax.cpu().numpy().astype(np.float64), ref["kept_vmax"]
    assert (vm >= rvm * (1 - 1e-7)).all() and (vm <= rvm * (1 + RADIUS_RTOL)).all()
    # real slots bit-exact; the tail and summary slots (rounded from double-float
    # sums on the GPU, from float64 in the oracle) within one bf16 step
    real = got["positions"] >= 0
    for x in ("pk", "pv"):
        assert (got[x][real] == ref[x][real]).all()
        dg = got[x][~real].astype(np.int32) - ref[x][~real].astype(np.int32)
        assert np.abs(dg).max() <= 1


@pytest.mark.parametrize("wl", sorted(WLS))
@pytest.mark.parametrize("m,tail_slot,qscale", [(3, 1, 1.0), (4, 0, 1.0), (3, 1, 1 / 64),
                                                (8, 0, 1 / 64)])
def test_certified_decode(m, tail_slot, qscale, wl):
    """With Gaussian keys in d = 128 the rank-grouped clusters have key radii
    near 16, so unit-variance queries give logit radii far above 1 and the
    certificate does not hold (agreement with the oracle is still checked);
    queries scaled by 1/64 bring the radii below 1 and the bound must then
    cover the true error."""
    WL = WLS[wl]
    K, V, Q, params, packed, ref, host = _run(m, tail_slot, WL)
    q = (W.draw_decode_queries(WL, 0, device="cuda").float() * qscale).to(torch.bfloat16)
    out, bound, cert = ck.certkv_decode_certified(q, packed, hkv=WL.H)
    torch.cuda.synchronize()
    qb = parity.bits(q).reshape(WL.B * WL.L, WL.Hq, WL.d)
    G = WL.Hq // WL.H
    scale = 1.0 / np.sqrt(WL.d)
    ref_out = np.zeros((WL.B * WL.L, WL.Hq, WL.d))
    ref_bound = np.zeros((WL.B * WL.L, WL.Hq))
    ref_cert = np.zeros((WL.B * WL.L, WL.Hq), bool)
    bound_tol = np.zeros((WL.B * WL.L, WL.Hq))
    for bl in range(WL.B * WL.L):
        for qh in range(WL.Hq):
            u = bl * WL.H + qh // G
            off, b = int(ref["offsets"][u]), int(ref["counts"][u])
            s0 = off + b + tail_slot
            o, bd, c, _ = oracle.decode_certified(
                qb[bl, qh], ref["pk"][off:off + b], ref["pv"][off:off + b], ref["pk"][s0:s0 + m],
                ref["pv"][s0:s0 + m], ref["cl_meta"][u, :m, 0].astype(np.int32),
                ref["cl_meta"][u, :m, 1], ref["cl_meta"][u, :m, 2], scale=scale)
            ref_out[bl, qh], ref_bound[bl, qh], ref_cert[bl, qh] = o, bd, c
            # The bound 3/Z (D_N + V'max D_Z) depends on the radii through
            # e^r (e^r - 1) with r = scale ||q|| R_g: a relative change eps of
            # the radii (the GPU rounds them up by 1e-5 and sums their squares
            # in fp32) changes the bound by at most (2 + 2 r) eps relative;
            # the cluster logits, norms and Z in fp32 add a few 1e-5.
            qf64 = oracle.bf16_bits_to_f64(qb[bl, qh])
            r_max = scale * np.linalg.norm(qf64) * ref["cl_meta"][u, :m, 1].max()
            bound_tol[bl, qh] = 3e-5 * (2.0 + 2.0 * r_max) + 6e-5
    parity.check_decode(out.reshape(WL.B * WL.L, WL.Hq, WL.d), ref_out)
    gb = bound.cpu().numpy().reshape(ref_bound.shape).astype(np.float64)
    # the bound is returned as fp32: beyond its range (a cluster with a strong
    # key and a unit query reaches e^(2r) of 1e70 and more) it is +inf
    big = ref_bound > np.finfo(np.float32).max
    assert np.isinf(gb[big]).all()
    rel = np.abs(gb[~big] - ref_bound[~big]) / np.maximum(np.abs(ref_bound[~big]), 1e-300)
    assert (rel <= bound_tol[~big]).all(), (float(rel.max()), float((rel / bound_tol[~big]).max()))
    assert (cert.cpu().numpy().reshape(ref_cert.shape).astype(bool) == ref_cert).all()
    # the bound against exact attention over every original token (float64)
    Kf = oracle.bf16_bits_to_f64(host["K"]).reshape(WL.B * WL.L, WL.H, WL.n, WL.d)
    Vf = oracle.bf16_bits_to_f64(host["V"]).reshape(WL.B * WL.L, WL.H, WL.n, WL.d)
    qf = oracle.bf16_bits_to_f64(qb)
    got = out.float().cpu().numpy().reshape(ref_out.shape)
    held = 0
    for bl in range(WL.B * WL.L):
        for qh in range(WL.Hq):
            if not ref_cert[bl, qh]:
                continue
            h = qh // G
            lg = scale * (Kf[bl, h] @ qf[bl, qh])
            w = np.exp(lg - lg.max())
            exact = (w[:, None] * Vf[bl, h]).sum(0) / w.sum()
            # the estimator itself (float64) is within the bound; the bf16 output adds its rounding
            assert np.linalg.norm(ref_out[bl, qh] - exact) <= ref_bound[bl, qh]
            assert np.linalg.norm(got[bl, qh] - exact) <= gb[bl, qh] + 2 ** -8 * np.linalg.norm(exact)
            held += 1
    if qscale < 1.0:
        assert held > 0
