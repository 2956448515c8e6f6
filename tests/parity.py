"""Comparison helpers for the CUDA-path-versus-oracle parity tests.

Tolerances (stated once, used by every parity test):
  * scores a, tail masses m and the fp32 tail centroids k*, v*: 1e-4 relative
    (scores per element; centroids relative to the vector's largest entry);
  * order, budgets, selected positions and packed real-slot bytes: bit-exact
    when the oracle starts from the GPU's own fp32 scores (conditioned mode);
  * from raw inputs (end-to-end mode) a budget may differ only as a certified
    near-tie of the allocation objective (relative gap <= 1e-6 under the
    oracle's curves), or where the order itself has a near-tie: scores that
    differ by less than 1e-6 relative in float64 can be equal in fp32, whose
    order (ties to the lower index) is then an equally valid order of the
    float64 scores; there the GPU's order must be a descending order of the
    float64 scores up to such near-ties, and the conditioned check certifies
    its budgets on that order.  A kept set may differ only by tokens whose
    score lies within 1e-6 relative of the cut;
  * decode outputs (bf16): 2e-2 maximum absolute error plus half a bf16 ulp
    of the reference value (the output is a bf16 number: rounding the exact
    result to bf16 alone moves it by up to half an ulp, 2^-5 at |o| = 8).
"""
from __future__ import annotations

import numpy as np

import oracle

RTOL_MASS = 1e-4
CUT_RTOL = 1e-6
OBJ_RTOL = 1e-6
ORDER_RTOL = 1e-6
DECODE_ATOL = 2e-2


def bits(t) -> np.ndarray:
    """uint16 view of a bf16 torch tensor, on the host."""
    import torch
    return t.detach().contiguous().cpu().view(torch.int16).numpy().view(np.uint16)


def check_scores(a_gpu: np.ndarray, a_ref: np.ndarray, rtol=RTOL_MASS):
    a_gpu = np.asarray(a_gpu, np.float64)
    rel = np.abs(a_gpu - a_ref) / np.maximum(np.abs(a_ref), 1e-300)
    worst = float(rel.max())
    assert worst <= rtol, f"score relative error {worst:.3e} > {rtol}"
    return worst


def packed_np(packed) -> dict:
    """Host copies of a Packed cache (numpy)."""
    d = dict(counts=packed.real_counts.cpu().numpy(), offsets=packed.offsets.cpu().numpy(),
             positions=packed.positions.cpu().numpy(), pk=bits(packed.k), pv=bits(packed.v))
    if packed.tail_f32 is not None:
        d["tail"] = packed.tail_f32.cpu().numpy().astype(np.float64)
        d["tail_mass"] = packed.tail_mass.cpu().numpy()
    return d


def slice_bl(p: dict, bl: int, H: int, B_live: int) -> dict:
    """The (sequence, layer) block bl of a packed cache, offsets rebased to 0."""
    s0, s1 = bl * B_live, (bl + 1) * B_live
    d = dict(counts=p["counts"][bl * H:(bl + 1) * H],
             offsets=np.concatenate([p["offsets"][bl * H:(bl + 1) * H] - s0, [B_live]]),
             positions=p["positions"][s0:s1], pk=p["pk"][s0:s1], pv=p["pv"][s0:s1])
    if "tail" in p:
        d["tail"] = p["tail"][bl * H:(bl + 1) * H]
        d["tail_mass"] = p["tail_mass"][bl * H:(bl + 1) * H]
    return d


def check_conditioned(got: dict, ref: dict, units: int, tail_slot: int = 1):
    """Bit-exact budgets / offsets / positions / real slots; tail within 1e-4."""
    counts, offsets, pos = got["counts"], got["offsets"], got["positions"]
    pk, pv = got["pk"], got["pv"]
    np.testing.assert_array_equal(counts, ref["counts"], err_msg="budgets differ")
    np.testing.assert_array_equal(offsets, ref["offsets"], err_msg="offsets differ")
    for u in range(units):
        o, c = int(offsets[u]), int(counts[u])
        np.testing.assert_array_equal(pos[o:o + c], ref["positions"][o:o + c],
                                      err_msg=f"kept positions differ (unit {u})")
        assert (pk[o:o + c] == ref["pk"][o:o + c]).all(), f"packed K differs (unit {u})"
        assert (pv[o:o + c] == ref["pv"][o:o + c]).all(), f"packed V differs (unit {u})"
        if tail_slot:
            assert pos[o + c] == -1
    worst = 0.0
    if tail_slot and "tail" in got:
        for u in range(units):
            for k in range(2):
                ref_v = ref["tail"][u, k]
                err = np.abs(got["tail"][u, k] - ref_v).max() / max(np.abs(ref_v).max(), 1e-300)
                worst = max(worst, err)
        assert worst <= RTOL_MASS, f"tail centroid relative error {worst:.3e}"
        merr = np.abs(got["tail_mass"] - ref["tail_mass"]) / np.maximum(ref["tail_mass"], 1e-300)
        assert merr.max() <= RTOL_MASS, f"tail mass relative error {merr.max():.3e}"
        # the packed tail slot is the bf16 rounding of the centroid: within half
        # a bf16 ulp of the value plus the 1e-4-of-the-vector centroid tolerance
        for u in range(units):
            s = int(offsets[u]) + int(counts[u])
            for arr, k in ((pk, 0), (pv, 1)):
                gv = oracle.bf16_bits_to_f64(arr[s])
                rv = ref["tail"][u, k]
                bound = np.abs(rv) * 2.0 ** -8 + RTOL_MASS * np.abs(rv).max()
                assert (np.abs(gv - rv) <= bound).all(), f"tail slot rounding (unit {u})"
    return worst


def gpu_order(a_gpu_u: np.ndarray) -> np.ndarray:
    """The order the CUDA path sorts into: its fp32 scores descending, equal
    values by lower index."""
    idx = np.arange(a_gpu_u.shape[0])
    return np.lexsort((idx, -np.asarray(a_gpu_u, np.float64)))


def order_near_tie(perm_gpu: np.ndarray, perm_ref: np.ndarray, a_ref_u: np.ndarray) -> bool:
    """True when the two orders differ and the first is nevertheless a
    descending order of the float64 scores up to near-ties (each adjacent pair
    out of float64 order within ORDER_RTOL relative)."""
    if np.array_equal(perm_gpu, perm_ref):
        return False
    s = a_ref_u[perm_gpu]
    drop = s[1:] - s[:-1]  # > 0 where the GPU order rises in float64
    return bool((drop <= ORDER_RTOL * np.maximum(np.abs(s[1:]), 1e-300)).all())


def check_end_to_end(got: dict, ref: dict, a_gpu: np.ndarray, H: int):
    """Budgets equal or certified near-ties; kept sets equal up to near-cut swaps.

    Returns the number of certified near-tie budget differences (of the
    objective or of the order)."""
    counts, offsets, pos = got["counts"], got["offsets"], got["positions"]
    units = counts.shape[0]
    near_ties = 0
    for bl in range(units // H):
        sl = slice(bl * H, (bl + 1) * H)
        if (counts[sl] != ref["counts"][sl]).any():
            cur = ref["c"][sl]
            obj_gpu = sum(cur[h, counts[bl * H + h]] for h in range(H))
            obj_ref = sum(cur[h, ref["counts"][bl * H + h]] for h in range(H))
            gap = abs(obj_gpu - obj_ref) / max(abs(obj_ref), 1e-300)
            assert counts[sl].sum() == ref["counts"][sl].sum()
            if gap > OBJ_RTOL:
                heads = range(bl * H, (bl + 1) * H)
                ties = [order_near_tie(gpu_order(a_gpu[u]), ref["perm"][u], ref["a"][u])
                        for u in heads]
                valid = all(np.array_equal(gpu_order(a_gpu[u]), ref["perm"][u]) or t
                            for u, t in zip(heads, ties))
                assert any(ties) and valid, \
                    f"budget mismatch in (seq,layer) {bl}: gap {gap:.3e} with no order near-tie"
            near_ties += 1
    for u in range(units):
        o, c = int(offsets[u]), int(counts[u])
        got_set = set(pos[o:o + c].tolist())
        want = set(oracle.select(ref["perm"][u], c).tolist())
        diff = got_set ^ want
        if diff:
            a = a_gpu[u].astype(np.float64)
            cut = np.sort(a)[::-1][c - 1]
            bad = [j for j in diff if abs(a[j] - cut) > CUT_RTOL * cut]
            assert not bad, f"unit {u}: kept-set swaps away from the cut: {bad[:5]}"
    return near_ties


def half_ulp_bf16(x) -> np.ndarray:
    """Half the bf16 unit in the last place at |x| (2^(e-8) for |x| in
    [2^e, 2^(e+1)); the subnormal quantum's half below 2^-126; 0 at 0)."""
    ax = np.abs(np.asarray(x, np.float64))
    _, e = np.frexp(np.maximum(ax, 2.0 ** -126))  # ax = f 2^e, f in [0.5, 1)
    return np.where(ax > 0, np.ldexp(1.0, e - 9), 0.0)


def check_decode(out, ref_out):
    """|got - oracle| <= 2e-2 + half a bf16 ulp of the oracle's value, element
    by element: the 2e-2 absolute bound of the parity contract, plus the
    rounding of the exact output to a bf16 number, which no implementation
    that returns bf16 can avoid."""
    got = out.float().cpu().numpy()
    tol = DECODE_ATOL + half_ulp_bf16(ref_out)
    err = np.abs(got - ref_out) - tol
    i = np.unravel_index(int(np.argmax(err)), err.shape)
    worst = float(np.abs(got - ref_out)[i])
    assert err[i] <= 0.0, (f"decode error {worst:.3e} at {i} above {tol[i]:.3e}: "
                           f"got {got[i]:.6g}, oracle {ref_out[i]:.6g}")
    return float(np.abs(got - ref_out).max())
