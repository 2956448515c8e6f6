"""Full-size workloads, in the launch configuration the benchmark times (every
layer and sequence in one call), checked against the oracle on sampled
(sequence, layer) blocks: conditioned mode bit-exact; end-to-end mode (the
oracle from the raw bf16 inputs) with scores within 1e-4, budgets equal or
certified near-ties and kept sets equal up to near-cut swaps; decode within
the decode tolerance; and the exact-budget equalities on every block."""
import numpy as np
import pytest
import torch

import oracle
import parity
from paper_2608_21541_gb300 import certkv as ck
from paper_2608_21541_gb300 import workloads as W

pytestmark = pytest.mark.gpu

# (workload, keep, sequence, layer) -> budget differences certified as near-ties
NEAR_TIES = {}


def _layer_host(K, V, Q, b, l):
    return (parity.bits(K[b:b + 1, l:l + 1]), parity.bits(V[b:b + 1, l:l + 1]),
            parity.bits(Q[b:b + 1, l:l + 1]))


def _check_blocks(wl, K, V, Q, a, packed, B_live, samples, e2e_scores=()):
    got = parity.packed_np(packed)
    H = wl.H
    cnt = got["counts"].reshape(wl.B * wl.L, H)
    assert (cnt.sum(1) == B_live - H).all(), "exact budget violated"
    assert got["offsets"][-1] == wl.B * wl.L * B_live
    a_host = a.view(wl.B, wl.L, H, wl.n)
    for (b, l) in samples:
        kb, vb, qb = _layer_host(K, V, Q, b, l)
        a_bl = a_host[b, l].cpu().numpy()
        kw = dict(B=1, L=1, Hq=wl.Hq, H=H, n=wl.n, d=wl.d, w=wl.w, B_live=B_live)
        ref = oracle.compress(kb, vb, None, a_in=a_bl, **kw)
        bl = b * wl.L + l
        block = parity.slice_bl(got, bl, H, B_live)
        parity.check_conditioned(block, ref, H)
        if (b, l) in e2e_scores:
            full = oracle.compress(kb, vb, qb, **kw)
            worst = parity.check_scores(a_bl, full["a"])
            ties = parity.check_end_to_end(block, full, a_bl, H)
            NEAR_TIES[(wl.name, wl.keep, b, l)] = ties
            print(f"{wl.name} keep {wl.keep} block ({b}, {l}): end-to-end score error "
                  f"{worst:.2e}, certified near-tie budgets {ties}")
    return got


def _run(wl, B_live, samples, e2e_scores=(), decode_steps=0, inputs=None):
    K, V, Q = inputs if inputs is not None else W.draw(wl, device="cuda")
    a = ck.certkv_score(K, Q)
    packed = ck.certkv_compress(K, V, Q, B_live, with_tail=True)
    torch.cuda.synchronize()
    got = _check_blocks(wl, K, V, Q, a, packed, B_live, samples, e2e_scores)
    for step in range(decode_steps):
        q = W.draw_decode_queries(wl, step, device="cuda")
        out = ck.certkv_decode_attn(q, packed, hkv=wl.H)
        for (b, l) in samples:
            bl = b * wl.L + l
            sub = parity.slice_bl(got, bl, wl.H, B_live)
            ref = oracle.decode(parity.bits(q[b:b + 1, l:l + 1]), sub["pk"], sub["pv"],
                                sub["offsets"], sub["counts"], B=1, L=1, Hq=wl.Hq, H=wl.H,
                                d=wl.d)
            parity.check_decode(out[b:b + 1, l:l + 1], ref)
    del a, packed
    if inputs is None:
        del K, V, Q
    torch.cuda.empty_cache()


def test_c2_full():
    wl = W.WORKLOADS["C2"]
    _run(wl, wl.B_live, samples=[(0, 0), (0, 13), (0, 31)], e2e_scores=[(0, 0)],
         decode_steps=1)


def test_c3_full():
    wl = W.WORKLOADS["C3"]
    _run(wl, wl.B_live, samples=[(0, 0), (0, 31)], e2e_scores=[(0, 0)], decode_steps=1)


def test_c4_full_with_decode():
    wl = W.WORKLOADS["C4"]
    _run(wl, wl.B_live, samples=[(0, 0), (7, 31)], e2e_scores=[(7, 31)], decode_steps=2)


def test_c5_full_budget_sweep():
    base = W.WORKLOADS["C5"]
    inputs = W.draw(base, device="cuda")
    for keep in base.keep_sweep:
        wl = base.with_(keep=keep)
        _run(wl, wl.B_live, samples=[(0, 0), (0, 79)], e2e_scores=[(0, 79)], decode_steps=1,
             inputs=inputs)


def test_context_of_2_20_tokens():
    """A 1048576-token context (one layer, 8 KV heads, 32 query heads, budget
    1/10), beyond the benchmark configurations: 512 sort tiles, 8192
    dispersion chunks and 4096 hull segments per head; at about ten hull
    candidates per group of eight segments (as at 131072 tokens) a layer has
    some 40 k candidates, more than the 12288 the allocator stages in shared
    memory, so its global-memory path runs.  Conditioned mode bit-exact on the
    layer, decode within its tolerance."""
    wl = W.Workload("L20", B=1, L=1, Hq=32, H=8, n=1 << 20, d=128, w=64, keep=(1, 10),
                    kind="zipf", description="2^20-token context")
    _run(wl, wl.B_live, samples=[(0, 0)], decode_steps=1)


def test_context_of_2_24_tokens():
    """The largest context the C ABI accepts: 16777216 tokens for 2 KV heads
    (4 query heads, budget 1/10; K and V 17 GB).  Byte offsets within a head
    reach 2^32 and the packed cache holds 3.4 M slots: conditioned mode
    bit-exact, decode within its tolerance."""
    wl = W.Workload("L24", B=1, L=1, Hq=4, H=2, n=1 << 24, d=128, w=32, keep=(1, 10),
                    kind="zipf", description="2^24-token context")
    _run(wl, wl.B_live, samples=[(0, 0)], decode_steps=1)
