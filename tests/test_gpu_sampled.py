"""Sampled tail compensation on the GPU against the float64 oracle, head by
head: the uniform-subset draws bit for bit (integer decisions taken in float64
on both sides), the weight-proportional draws equal or certified near-ties of
the oracle's own cumulative tail weight, and every statistic, given the GPU's
draws, within floating-point tolerance; small cases and sampled heads of the
full 131072-token workload."""
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


def _f64(b):
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def _run(wl, m, layers=None, seed=11):
    K, V, Q = W.draw(wl, device="cuda", layers=layers)
    packed = ck.certkv_compress(K, V, Q, wl.B_live)
    q = W.draw_decode_queries(wl, 0, device="cuda", layers=layers)
    B, L = q.shape[0], q.shape[1]
    g = torch.Generator().manual_seed(seed)
    unif = torch.rand((B, L, wl.Hq, 2 * m), generator=g, dtype=torch.float32)
    stats, idx = ck.certkv_sampled_compensation(q, K, V, packed, unif.cuda(), m)
    torch.cuda.synchronize()
    BL = B * L
    return dict(
        BL=BL, stats=stats.cpu().numpy().astype(np.float64).reshape(BL, wl.Hq, 8),
        idx=idx.cpu().numpy().reshape(BL, wl.Hq, 2 * m), unif=unif.numpy().reshape(BL, wl.Hq, 2 * m),
        Kb=parity.bits(K).reshape(BL, wl.H, wl.n, wl.d), Vb=parity.bits(V).reshape(BL, wl.H, wl.n, wl.d),
        qb=parity.bits(q).reshape(BL, wl.Hq, wl.d), pos=packed.positions.cpu().numpy(),
        offs=packed.offsets.cpu().numpy(), cnts=packed.real_counts.cpu().numpy())


def _check_head(r, wl, bl, qh, m):
    G = wl.Hq // wl.H
    h = qh // G
    u = bl * wl.H + h
    scale = 1.0 / math.sqrt(wl.d)
    kept = np.zeros(wl.n, bool)
    kept[r["pos"][r["offs"][u]:r["offs"][u] + r["cnts"][u]]] = True
    uu = r["unif"][bl, qh]
    gidx, gst = r["idx"][bl, qh], r["stats"][bl, qh]
    ref_idx, _ = oracle.sampled_compensation(r["qb"][bl, qh], r["Kb"][bl, h], r["Vb"][bl, h], kept,
                                             uu, scale=scale, m=m)
    tag = (bl, qh)
    np.testing.assert_array_equal(gidx[m:], ref_idx[m:], err_msg=f"uniform subset {tag}")
    # weight-proportional draws: equal, or the oracle's cumulative weight puts
    # the target within 1e-6 of the GPU's token's interval
    z = scale * (_f64(r["Kb"][bl, h]) @ _f64(r["qb"][bl, qh]))
    w = np.where(kept, 0.0, np.exp(z - z.max()))
    cum = np.cumsum(w)
    for k in range(m):
        if gidx[k] != ref_idx[k]:
            j = int(gidx[k])
            target = float(uu[k]) * cum[-1]
            assert not kept[j], ("drew a kept token", tag, k, j)
            lo = cum[j] - w[j]
            assert lo <= target + 1e-6 * cum[-1] and cum[j] >= target - 1e-6 * cum[-1], \
                ("weighted draw not a near-tie", tag, k, j, int(ref_idx[k]))
    # statistics given the GPU's draws
    _, st = oracle.sampled_compensation(r["qb"][bl, qh], r["Kb"][bl, h], r["Vb"][bl, h], kept, uu,
                                        scale=scale, m=m, forced_idx=gidx)
    assert abs(gst[0] - st[0]) <= 1e-5 * st[0] + 1e-7, ("p_S", tag, gst[0], st[0])
    for i in (1, 2, 5, 6, 7):
        assert abs(gst[i] - st[i]) <= 2e-4 * abs(st[i]) + 1e-7, (i, tag, gst[i], st[i])
    for i in (3, 4):
        assert abs(gst[i] - st[i]) <= 1e-4 * st[2] + 1e-6, (i, tag, gst[i], st[i])


@pytest.mark.parametrize("name", sorted(CASES))
def test_sampled_compensation_matches_oracle(name):
    wl, m = CASES[name], 8
    r = _run(wl, m)
    for bl in range(r["BL"]):
        for qh in range(wl.Hq):
            _check_head(r, wl, bl, qh, m)


def test_sampled_compensation_full_size_sampled():
    """One layer of the 131072-token workload, eight sampled query heads, m = 32."""
    wl, m = W.WORKLOADS["C3"], 32
    r = _run(wl, m, layers=[3])
    rng = np.random.default_rng(5)
    for qh in rng.choice(wl.Hq, size=8, replace=False):
        _check_head(r, wl, 0, int(qh), m)
