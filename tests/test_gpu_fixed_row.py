"""Fixed-row diagnostics (Theorem: fixed-row tail factorization) on the GPU
against the float64 oracle, head by head, for the compressed caches of the
small cases; and the theorem's inequality on every head."""
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
}


@pytest.mark.parametrize("name", sorted(CASES))
@pytest.mark.parametrize("tail_slot", [1, 0])
def test_fixed_row_stats_match_oracle(name, tail_slot):
    wl = CASES[name]
    K, V, Q = W.draw(wl, device="cuda")
    params = ck.certkv_default_params(tail_slot=tail_slot)
    packed = ck.certkv_compress(K, V, Q, wl.B_live, params)
    q = W.draw_decode_queries(wl, 0, device="cuda")
    out = ck.certkv_decode_attn(q, packed, hkv=wl.H)
    stats = ck.certkv_fixed_row_stats(q, K, V, packed)
    torch.cuda.synchronize()
    got = stats.cpu().numpy().astype(np.float64).reshape(wl.B * wl.L, wl.Hq, 8)
    Kb = parity.bits(K).reshape(wl.B * wl.L, wl.H, wl.n, wl.d)
    Vb = parity.bits(V).reshape(wl.B * wl.L, wl.H, wl.n, wl.d)
    qb = parity.bits(q).reshape(wl.B * wl.L, wl.Hq, wl.d)
    oh = out.float().cpu().numpy().astype(np.float64).reshape(wl.B * wl.L, wl.Hq, wl.d)
    pos = packed.positions.cpu().numpy()
    offs = packed.offsets.cpu().numpy()
    cnts = packed.real_counts.cpu().numpy()
    G = wl.Hq // wl.H
    scale = 1.0 / np.sqrt(wl.d)
    for bl in range(wl.B * wl.L):
        for qh in range(wl.Hq):
            h = qh // G
            u = bl * wl.H + h
            kept = np.zeros(wl.n, bool)
            kept[pos[offs[u]:offs[u] + cnts[u]]] = True
            ref = oracle.fixed_row(qb[bl, qh], Kb[bl, h], Vb[bl, h], kept, scale=scale,
                                   ohat=oh[bl, qh])
            g = got[bl, qh]
            assert abs(g[0] - ref[0]) <= 1e-5 * ref[0] + 1e-7, ("kept mass", g[0], ref[0])
            for i in (1, 3, 4, 6):
                assert abs(g[i] - ref[i]) <= 1e-4 * abs(ref[i]) + 1e-6, (i, g[i], ref[i])
            for i in (2, 5):  # errors: absolute, relative to the output's scale
                assert abs(g[i] - ref[i]) <= 1e-4 * ref[1] + 1e-6, (i, g[i], ref[i])
            assert g[7] <= 1e-4 * ref[1] + 1e-6
            assert g[2] <= g[4] * (1 + 1e-5) + 1e-6  # the theorem's mass bound
