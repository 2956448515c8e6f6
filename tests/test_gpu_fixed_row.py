"""Fixed-row diagnostics on the GPU against the float64 oracle, head by head:
the fixed-row tail factorization quantities (fields 0-7) and the future-query
lift quantities (fields 8-15), for the compressed caches of small cases and a
sampled layer at the full C3 size; and the two theorems' inequalities on every
head."""
import math

import numpy as np
import pytest
import torch

import oracle
import parity
from paper_2608_21541_gb300 import certkv as ck
from paper_2608_21541_gb300 import workloads as W

pytestmark = pytest.mark.gpu

CASES = {
    "planted_g4": W.Workload("S", B=2, L=2, Hq=8, H=2, n=3000, d=128, w=20, keep=(1, 10),
                             kind="planted"),
    "zipf_g8": W.Workload("Z", B=1, L=1, Hq=16, H=2, n=5000, d=128, w=32, keep=(1, 5),
                          kind="zipf"),
    # tiny contexts: every tile of the instrument ragged; tails of 20 tokens or more
    "tiny33_g16": W.Workload("T33", B=1, L=2, Hq=16, H=1, n=33, d=128, w=3, keep=(1, 3),
                             kind="zipf"),
    "tiny64_h3": W.Workload("T64", B=1, L=1, Hq=12, H=3, n=64, d=128, w=4, keep=(1, 4),
                            kind="zipf"),
}
NF = len(ck.FIXED_ROW_FIELDS)


def _run(wl, tail_slot, layers=None):
    K, V, Q = W.draw(wl, device="cuda", layers=layers)
    L = K.shape[1]
    params = ck.certkv_default_params(tail_slot=tail_slot)
    packed = ck.certkv_compress(K, V, Q, wl.B_live, params)
    scores = ck.certkv_score(K, Q, params)
    q = W.draw_decode_queries(wl, 0, device="cuda", layers=layers)
    out = ck.certkv_decode_attn(q, packed, hkv=wl.H)
    stats = ck.certkv_fixed_row_stats(q, K, V, packed, scores=scores)
    bare = ck.certkv_fixed_row_stats(q, K, V, packed)
    torch.cuda.synchronize()
    BL = wl.B * L
    return dict(
        L=L, BL=BL,
        got=stats.cpu().numpy().astype(np.float64).reshape(BL, wl.Hq, NF),
        bare=bare.cpu().numpy().astype(np.float64).reshape(BL, wl.Hq, NF),
        Kb=parity.bits(K).reshape(BL, wl.H, wl.n, wl.d),
        Vb=parity.bits(V).reshape(BL, wl.H, wl.n, wl.d),
        qb=parity.bits(q).reshape(BL, wl.Hq, wl.d),
        oh=out.float().cpu().numpy().astype(np.float64).reshape(BL, wl.Hq, wl.d),
        a=scores.cpu().numpy().reshape(BL, wl.H, wl.n),
        pos=packed.positions.cpu().numpy(), offs=packed.offsets.cpu().numpy(),
        cnts=packed.real_counts.cpu().numpy(),
        pk=parity.bits(packed.k), pv=parity.bits(packed.v))


def _check_head(r, wl, bl, qh, tail_slot):
    G = wl.Hq // wl.H
    h = qh // G
    u = bl * wl.H + h
    scale = 1.0 / math.sqrt(wl.d)
    kept = np.zeros(wl.n, bool)
    kept[r["pos"][r["offs"][u]:r["offs"][u] + r["cnts"][u]]] = True
    ref = oracle.fixed_row(r["qb"][bl, qh], r["Kb"][bl, h], r["Vb"][bl, h], kept, scale=scale,
                           ohat=r["oh"][bl, qh])
    srow = r["offs"][u] + r["cnts"][u]
    ks = r["pk"][srow] if tail_slot else None
    vs = r["pv"][srow] if tail_slot else None
    lift = oracle.future_query_lift(r["qb"][bl, qh], r["Kb"][bl, h], r["Vb"][bl, h], kept,
                                    r["a"][bl, h], scale=scale, kstar=ks, vstar=vs)
    g = r["got"][bl, qh]
    tag = (bl, qh)
    # fixed-row tail factorization
    assert abs(g[0] - ref[0]) <= 1e-5 * ref[0] + 1e-7, ("kept mass", tag, g[0], ref[0])
    for i in (1, 3, 4, 6):
        assert abs(g[i] - ref[i]) <= 1e-4 * abs(ref[i]) + 1e-6, (i, tag, g[i], ref[i])
    for i in (2, 5):  # errors: absolute, relative to the output's scale
        assert abs(g[i] - ref[i]) <= 1e-4 * ref[1] + 1e-6, (i, tag, g[i], ref[i])
    assert g[7] <= 1e-4 * ref[1] + 1e-6
    assert g[2] <= g[4] * (1 + 1e-5) + 1e-6  # the mass bound
    # future-query lift
    assert abs(g[8] - lift[0]) <= 1e-5 * lift[0] + 1e-7, ("tail mass", tag, g[8], lift[0])
    assert abs(g[9] - lift[1]) <= 1e-5, ("slot weight", tag, g[9], lift[1])
    for i in (10, 14):  # L1 sums of weights in [0, 2]
        assert abs(g[i] - lift[i - 8]) <= 1e-4 * lift[i - 8] + 2e-5, (i, tag, g[i], lift[i - 8])
    assert abs(g[12] - lift[4]) <= 1e-4 * lift[4] + 2e-5 * g[6], ("lift bound", tag, g[12], lift[4])
    if tail_slot:
        assert abs(g[11] - lift[3]) <= 1e-4 * (1 + abs(lift[3])), ("gap", tag, g[11], lift[3])
        assert abs(g[13] - lift[5]) <= 1e-5, ("tanh bound", tag, g[13], lift[5])
        assert abs(g[15] - lift[7]) <= 1e-5 + 1e-4 * lift[7], ("mixture", tag, g[15], lift[7])
        # |p - q| <= tanh(|Lambda_T - z*| / 4)
        assert abs(g[8] - g[9]) <= g[13] + 1e-5
    else:
        assert g[9] == 0.0 and all(math.isnan(g[i]) for i in (11, 13, 15))
    # ||O - O-hat|| <= V_max ||A - Abar||_1 + q ||v* - mixture||, up to the bf16
    # rounding of the decode output (half an ulp per coordinate)
    slack = 2.0 ** -8 * (ref[1] + g[5]) + 1e-5
    mix = g[15] if tail_slot else 0.0
    assert g[5] <= g[6] * g[14] + g[9] * mix + slack, ("lift inequality", tag)
    assert g[14] <= 2 * abs(g[8] - g[9]) + min(g[8], g[9]) * g[10] + 1e-5
    # without scores: the r-dependent fields are NaN, the rest unchanged
    b = r["bare"][bl, qh]
    for i in range(NF):
        if i in (10, 12, 14, 15):
            assert math.isnan(b[i]), (i, tag)
        elif not math.isnan(g[i]):
            assert b[i] == g[i], (i, tag, b[i], g[i])


@pytest.mark.parametrize("name", sorted(CASES))
@pytest.mark.parametrize("tail_slot", [1, 0])
def test_fixed_row_stats_match_oracle(name, tail_slot):
    wl = CASES[name]
    r = _run(wl, tail_slot)
    for bl in range(r["BL"]):
        for qh in range(wl.Hq):
            _check_head(r, wl, bl, qh, tail_slot)


def test_fixed_row_stats_full_size_sampled():
    """One layer of the 131072-token workload, eight sampled query heads."""
    wl = W.WORKLOADS["C3"]
    r = _run(wl, 1, layers=[5])
    rng = np.random.default_rng(7)
    for qh in rng.choice(wl.Hq, size=8, replace=False):
        _check_head(r, wl, 0, int(qh), 1)
