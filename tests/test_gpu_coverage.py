"""Coverage profile on the GPU against the float64 oracle, row by row: the
logit at every rank, the ranked gap profile, the coverage budgets K_eta (equal,
or a near-tie that the oracle's own cumulative mass certifies), the relative
and calibrated counts (equal up to tokens within the logit tolerance of the
threshold), the maximum logit and the log-partition; the order's ties by lower
index; and sampled rows at the full 131072-token size."""
import math

import numpy as np
import pytest
import torch

import oracle
import parity
from paper_2608_21541_gb300 import certkv as ck
from paper_2608_21541_gb300 import workloads as W

pytestmark = pytest.mark.gpu

ETA = (0.5, 0.1, 0.05, 0.01)
REL = (0.5, 0.1, 0.01)
ABS = (0.01, 1e-3, 1e-4)
LOGIT_TOL = 5e-5  # fp32 logits of 128-term bf16 dot products, |z| of order 1-10


def _f64(b: np.ndarray) -> np.ndarray:
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


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
    "gauss_g4": W.WORKLOADS["C1"],
}


def _profile(K, q):
    r = ck.certkv_coverage_profile(q, K, eta=ETA, rel_eps=REL, abs_eps=ABS, with_order=True,
                                   with_gap=True)
    torch.cuda.synchronize()
    return {k: (v.cpu().numpy() if v is not None else None) for k, v in r.items()}


def _check_row(got, ref, zo, tag):
    """got: this row's GPU outputs; ref: the oracle's; zo: the oracle's logits
    in token order (float64)."""
    n = zo.size
    z_sorted = zo[ref["order"]]
    order = got["order"].astype(np.int64)
    assert np.array_equal(np.sort(order), np.arange(n)), ("order is not a permutation", tag)
    # the logit at each rank agrees whichever near-tied token sits there
    assert np.abs(zo[order] - z_sorted).max() <= LOGIT_TOL, ("order", tag)
    assert np.abs(got["gap"].astype(np.float64) - ref["gap"]).max() <= LOGIT_TOL, ("gap", tag)
    assert abs(got["top"][0] - ref["top"][0]) <= 1e-5 * (1 + abs(ref["top"][0])), ("max", tag)
    assert abs(got["top"][1] - ref["top"][1]) <= 1e-5 * (1 + abs(ref["top"][1])), ("lse", tag)
    w = np.exp(-ref["gap"])
    C = np.cumsum(w) / w.sum()
    for e, eta in enumerate(ETA):
        k = int(got["K_eta"][e])
        if k != ref["K_eta"][e]:  # a near-tie: the oracle's mass crosses 1 - eta within tolerance
            assert 1 <= k <= n, ("K_eta range", tag, eta, k)
            assert C[k - 1] >= 1 - eta - 2e-5, ("K_eta too small", tag, eta, k, ref["K_eta"][e])
            assert k == 1 or C[k - 2] < 1 - eta + 2e-5, ("K_eta too large", tag, eta, k)
    rel_margin = zo - ref["top"][0]
    for e, eps in enumerate(REL):
        lo = int((rel_margin - math.log(eps) > LOGIT_TOL).sum())
        hi = int((rel_margin - math.log(eps) > -LOGIT_TOL).sum())
        assert lo <= got["rel"][e] <= hi, ("relative count", tag, eps, got["rel"][e], ref["rel"][e])
    abs_margin = zo - ref["top"][1]
    for e, eps in enumerate(ABS):
        lo = int((abs_margin - math.log(eps) > LOGIT_TOL).sum())
        hi = int((abs_margin - math.log(eps) > -LOGIT_TOL).sum())
        assert lo <= got["abs"][e] <= hi, ("calibrated count", tag, eps, got["abs"][e], ref["abs"][e])


def _check_all(wl, K, q, rows=None):
    got = _profile(K, q)
    BL = K.shape[0] * K.shape[1]
    Kb = parity.bits(K).reshape(BL, wl.H, wl.n, wl.d)
    qb = parity.bits(q).reshape(BL, wl.Hq, wl.d)
    G = wl.Hq // wl.H
    scale = 1.0 / math.sqrt(wl.d)
    flat = {k: v.reshape(BL * wl.Hq, -1) for k, v in got.items()}
    rows = range(BL * wl.Hq) if rows is None else rows
    for row in rows:
        bl, qh = divmod(int(row), wl.Hq)
        ref = oracle.coverage_profile(qb[bl, qh], Kb[bl, qh // G], scale=scale, eta=ETA,
                                      rel_eps=REL, abs_eps=ABS)
        zo = scale * (_f64(Kb[bl, qh // G]) @ _f64(qb[bl, qh]))
        _check_row({k: v[row] for k, v in flat.items()}, ref, zo, (bl, qh))
    return flat


@pytest.mark.parametrize("name", sorted(CASES))
def test_coverage_profile_matches_oracle(name):
    wl = CASES[name]
    K, _, _ = W.draw(wl, device="cuda")
    q = W.draw_decode_queries(wl, 0, device="cuda")
    _check_all(wl, K, q)


def test_coverage_ties_by_lower_index():
    """Every odd token repeats the key of the even token before it, so the two
    logits are bit-identical on both sides: the lower index ranks first."""
    wl = CASES["planted_g4"]
    K, _, _ = W.draw(wl, device="cuda")
    K[..., 1::2, :] = K[..., 0::2, :]
    q = W.draw_decode_queries(wl, 0, device="cuda")
    flat = _check_all(wl, K, q)
    rank = np.empty_like(flat["order"])
    rows = np.arange(flat["order"].shape[0])[:, None]
    rank[rows, flat["order"]] = np.arange(wl.n)[None, :]
    assert (rank[:, 0::2] < rank[:, 1::2]).all()


def test_coverage_profile_full_size_sampled():
    """One layer of the 131072-token workload, eight sampled rows."""
    wl = W.WORKLOADS["C3"]
    K, _, _ = W.draw(wl, device="cuda", layers=[9])
    q = W.draw_decode_queries(wl, 0, device="cuda", layers=[9])
    rng = np.random.default_rng(3)
    _check_all(wl, K, q, rows=rng.choice(wl.Hq, size=8, replace=False))
