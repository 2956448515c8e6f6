"""Pins of the float64 oracle to what the paper and the mathematics fix.

Each ``pin_*`` function raises AssertionError when the oracle (or a variant
of it passed as ``lib``) disagrees with a value, identity, bound or brute-force
result that does not come from the oracle itself.  ``test_oracle_pins.py``
runs them on the oracle; ``test_oracle_mutations.py`` runs them on copies of
the oracle with a planted mistake and checks that some pin fails.
"""
from __future__ import annotations

import itertools
import json
import math
import os

import numpy as np
from scipy.special import softmax
from scipy.stats import norm

import oracle

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def golden(name: str) -> dict:
    with open(os.path.join(GOLDEN, "paper_examples.json")) as f:
        return json.load(f)[name]


def to_bf16_bits(x) -> np.ndarray:
    """float -> bf16 bit patterns, round to nearest even (via float32)."""
    f = np.ascontiguousarray(np.asarray(x, dtype=np.float32))
    u = f.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return u.astype(np.uint16)


def bf(x) -> np.ndarray:
    """float64 values of bf16 data: bit patterns (uint16) are widened exactly,
    anything else is first rounded to bf16."""
    x = np.asarray(x)
    if x.dtype == np.uint16:
        return oracle.bf16_bits_to_f64(x)
    return oracle.bf16_bits_to_f64(to_bf16_bits(x))


# ------------------------------------------------------------------ scores --

def pin_scores_softmax_row(lib=None):
    """With one observation row, one query head, no pooling and no window
    protection the score vector is exactly one softmax row (§4: the scorer sums
    softmax attention weights; a = s / sum s)."""
    rng = np.random.default_rng(1)
    n, d = 300, 16
    K = to_bf16_bits(rng.standard_normal((n, d)))
    q = to_bf16_bits(rng.standard_normal((1, 1, d)))
    scale = 0.37
    a = oracle.scores(K, q, w=1, G=1, scale=scale, pool=1, protect=0, lib=lib)
    ref = softmax(scale * (bf(K) @ bf(q)[0, 0]))
    np.testing.assert_allclose(a, ref, rtol=1e-12, atol=0)


def pin_scores_masked_rows(lib=None):
    """Mean of causally masked softmax rows over every (query head, window row)
    of the group (observation-window scorer, reading R-A1), no pooling."""
    rng = np.random.default_rng(2)
    n, d, w, G = 40, 8, 4, 3
    K = to_bf16_bits(rng.standard_normal((n, d)))
    Qg = to_bf16_bits(rng.standard_normal((G, w, d)))
    scale = 1 / math.sqrt(d)
    a = oracle.scores(K, Qg, w=w, G=G, scale=scale, pool=1, protect=0, lib=lib)
    Kf, Qf = bf(K), bf(Qg)
    s = np.zeros(n)
    for g in range(G):
        for t in range(w):
            logits = scale * (Kf @ Qf[g, t])
            logits[np.arange(n) > n - w + t] = -np.inf
            s += softmax(logits)
    np.testing.assert_allclose(a, s / s.sum(), rtol=1e-12, atol=0)


def pin_scores_pool_onehot(lib=None):
    """A score vector that is (numerically) one-hot at j0 pools into five
    equal entries of 1/5 (zero padding, divided by the width); the window keys
    get the maximum pooled score.  At j0 = 1 only four pooled entries survive,
    each 1/5, so a = 1/(4 + w) on them and on the window keys."""
    n, d, w = 30, 4, 3
    for j0, count in ((10, 5), (1, 4)):
        K = np.zeros((n, d))
        rng = np.random.default_rng(3)
        K[:] = 0.01 * rng.standard_normal((n, d))
        K[j0] = [8.0, 0, 0, 0]
        Qg = np.zeros((1, w, d))
        Qg[0, :, 0] = 8.0
        a = oracle.scores(to_bf16_bits(K), to_bf16_bits(Qg), w=w, G=1, scale=0.625,
                          pool=5, protect=1, lib=lib)
        lo = max(0, j0 - 2)
        hot = list(range(lo, j0 + 3))
        assert len(hot) == count
        expect = 1.0 / (count + w)
        np.testing.assert_allclose(a[hot], expect, rtol=1e-9)
        np.testing.assert_allclose(a[n - w:], expect, rtol=1e-9)
        cold = [j for j in range(n - w) if j not in hot]
        assert a[cold].max() < 1e-12


def pin_scores_probability(lib=None):
    """a_j >= 0 and sum_j a_j = 1 (implementation appendix: a = (s)_+ / sum (s)_+)."""
    rng = np.random.default_rng(4)
    n, d, w, G = 500, 32, 16, 4
    K = to_bf16_bits(rng.standard_normal((n, d)))
    Qg = to_bf16_bits(rng.standard_normal((G, w, d)))
    a = oracle.scores(K, Qg, w=w, G=G, scale=1 / math.sqrt(d), lib=lib)
    assert (a >= 0).all()
    assert abs(a.sum() - 1.0) < 1e-12


# ------------------------------------------------------------------- order --

def pin_order_brute_force(lib=None):
    """Descending score, ties broken by the lower index (the paper's convention
    for the order pi)."""
    rng = np.random.default_rng(5)
    a = rng.integers(0, 6, size=200) / 5.0
    perm = oracle.order(a, lib=lib)
    ref = sorted(range(a.size), key=lambda j: (-a[j], j))
    assert perm.tolist() == ref


def pin_topk_mass_optimal(lib=None):
    """Top-k by weight keeps the largest mass among all k-subsets (lemma
    'top-k is coverage-optimal'), checked by exhaustive search."""
    rng = np.random.default_rng(6)
    a = rng.dirichlet(np.ones(10))
    perm = oracle.order(a, lib=lib)
    for k in range(1, 10):
        best = max(sum(a[list(c)]) for c in itertools.combinations(range(10), k))
        assert abs(a[perm[:k]].sum() - best) < 1e-15
        kept = oracle.select(perm, k, lib=lib)
        assert kept.tolist() == sorted(perm[:k].tolist())


# ------------------------------------------------------------------ curves --

def _centred(a, Vf, perm, b):
    E = perm[b:]
    m = a[E].sum()
    vstar = (a[E, None] * Vf[E]).sum(0) / m
    S = (a[E] * ((Vf[E] - vstar) ** 2).sum(1)).sum()
    return m, vstar, S


def pin_curve_centred_definition(lib=None):
    """c(b) = sqrt(m(b) S(b)) with the centred second moment
    S = sum_E a_j ||v_j - v*||^2 computed directly (implementation appendix;
    Eq. certkv-curve), against the suffix-scan formula of the oracle; the
    uncentred and tail-mass statistics are sqrt(m Q) and m."""
    rng = np.random.default_rng(7)
    n, d = 12, 6
    a = rng.dirichlet(np.ones(n))
    a[3] = a[7]  # one tie
    a /= a.sum()
    V = to_bf16_bits(rng.standard_normal((n, d)) + 0.3)
    Vf = bf(V)
    perm = oracle.order(a, lib=lib)
    c0 = oracle.curve(a, V, perm, 0, lib=lib)
    c1 = oracle.curve(a, V, perm, 1, lib=lib)
    c2 = oracle.curve(a, V, perm, 2, lib=lib)
    for b in range(n):
        m, vstar, S = _centred(a, Vf, perm, b)
        Q = (a[perm[b:]] * (Vf[perm[b:]] ** 2).sum(1)).sum()
        assert abs(c0[b] - math.sqrt(m * S)) <= 1e-12 * max(1.0, c0[b]), (b, c0[b])
        assert abs(c1[b] - math.sqrt(m * Q)) <= 1e-12 * c1[b]
        assert abs(c2[b] - m) <= 1e-14


def pin_curve_envelope(lib=None):
    """Err_1(E(b)) = sum_E a_j ||v_j - v*|| <= c(b) (weighted Cauchy-Schwarz,
    Theorem 'exact dispersion envelopes' (b)) and the feasibility bound
    c(b)^2 <= m (Vmax^2 - ||v*||^2) of the same theorem."""
    rng = np.random.default_rng(8)
    n, d = 64, 8
    a = rng.dirichlet(np.full(n, 0.5))
    V = to_bf16_bits(rng.standard_normal((n, d)))
    Vf = bf(V)
    vmax2 = (Vf ** 2).sum(1).max()
    perm = oracle.order(a, lib=lib)
    c = oracle.curve(a, V, perm, 0, lib=lib)
    for b in range(n):
        m, vstar, _ = _centred(a, Vf, perm, b)
        E = perm[b:]
        err1 = (a[E] * np.sqrt(((Vf[E] - vstar) ** 2).sum(1))).sum()
        assert err1 <= c[b] * (1 + 1e-12) + 1e-15
        assert c[b] ** 2 <= m * (vmax2 - (vstar ** 2).sum()) * (1 + 1e-12) + 1e-15


def pin_curve_two_point_witness(lib=None):
    """The two-point tail v* +- delta u with equal weights attains
    Err_1 = sqrt(m S) = m delta (Theorem 'exact dispersion envelopes', proof of
    (b)); a single-token tail has zero dispersion."""
    a = np.array([0.5, 0.25, 0.25])
    V = np.zeros((3, 4))
    V[0] = [3.0, 1.0, -2.0, 0.5]
    V[1] = [1.0, 0.5, 0.0, 0.0]
    V[2] = [1.0, -0.5, 0.0, 0.0]
    perm = oracle.order(a, lib=lib)
    assert perm.tolist() == [0, 1, 2]
    c = oracle.curve(a, to_bf16_bits(V), perm, 0, lib=lib)
    assert abs(c[1] - 0.5 * 0.5) < 1e-15
    assert c[2] == 0.0


# -------------------------------------------------------------- allocation --

def pin_allocation_nonconvex_example(lib=None):
    """Hand-worked Algorithm 1 on a non-convex pair of curves (golden)."""
    g = golden("allocation_nonconvex")
    b, rep = oracle.allocate(np.array(g["curves"], float), g["B_real"], g["alpha_num"],
                             g["alpha_den"], 40, lib=lib)
    assert b.tolist() == g["expected_b"], b
    assert rep == 0
    bg, _ = oracle.allocate(np.array(g["curves"], float), g["B_real"], g["alpha_num"],
                            g["alpha_den"], 0, lib=lib)
    assert bg.tolist() == g["greedy_b"], bg


def _brute_force(curves, B_real, bmin):
    H, n = curves.shape
    best, arg = math.inf, None
    for bs in itertools.product(range(bmin, n), repeat=H):
        if sum(bs) != B_real:
            continue
        obj = sum(curves[h, bs[h]] for h in range(H))
        if obj < best:
            best, arg = obj, bs
    return best, arg


def pin_allocation_equalities_and_optimality(lib=None):
    """sum_h b_h = B_real and b_min <= b_h <= n - 1 (exact-budget protocol);
    for strictly convex curves the result equals the exhaustive optimum
    (separable convex integer allocation), and for non-convex curves it is
    never better than that optimum (the paper calls the allocator a heuristic)."""
    rng = np.random.default_rng(9)
    H, n = 3, 9
    for trial in range(12):
        if trial % 2 == 0:  # strictly convex, decreasing
            steps = -np.sort(rng.uniform(0.05, 1.0, size=(H, n - 1)), axis=1)[:, ::-1]
            curves = np.concatenate([np.full((H, 1), 10.0), 10.0 + np.cumsum(steps, 1)], 1)
        else:
            curves = rng.uniform(0, 5, size=(H, n))
        for B_real in (H, 7, 12, 17, H * (n - 1)):
            bmin = oracle.b_min(B_real, H, 1, 5, lib=lib)
            if B_real < H * bmin:
                continue
            b, _ = oracle.allocate(curves, B_real, 1, 5, 40, lib=lib)
            assert b.sum() == B_real
            assert (b >= bmin).all() and (b <= n - 1).all()
            best, arg = _brute_force(curves, B_real, bmin)
            obj = sum(curves[h, b[h]] for h in range(H))
            if trial % 2 == 0:
                assert list(b) == list(arg), (trial, B_real, b, arg)
            else:
                assert obj >= best - 1e-12


def pin_allocator_true_uniform(lib=None):
    """Allocator ablation "true uniform" (reading R-A15): the budget split as
    evenly as integers allow, the remainder to the lowest heads, whatever the
    curves."""
    rng = np.random.default_rng(21)
    for H, n, B_real in ((3, 9, 7), (4, 20, 40), (5, 6, 25), (2, 33, 2)):
        curves = rng.uniform(0, 5, size=(H, n))
        b, rep = oracle.allocate(curves, B_real, 1, 5, 40, mode=1, lib=lib)
        assert b.sum() == B_real and rep == 0
        assert b.max() - b.min() <= 1
        assert all(b[h] >= b[h + 1] for h in range(H - 1)), b  # extra tokens go to low heads


def pin_allocator_greedy_marginal(lib=None):
    """Allocator ablation "greedy marginal" (reading R-A16): from b_min, one
    token at a time to the smallest marginal.  For separable convex curves
    greedy marginal allocation is optimal (textbook resource allocation), so
    it must match the exhaustive optimum; on the hand-worked non-convex pair
    it takes c_0's two steepest marginals first, then the tie -0.5 / -0.5 goes
    to head 0: b = [4, 1] after 3 single-token steps."""
    rng = np.random.default_rng(5)
    H, n = 3, 8
    for _ in range(6):
        steps = -np.sort(rng.uniform(0.05, 1.0, size=(H, n - 1)), axis=1)[:, ::-1]
        curves = np.concatenate([np.full((H, 1), 10.0), 10.0 + np.cumsum(steps, 1)], 1)
        for B_real in (H, 8, 13, H * (n - 1)):
            bmin = oracle.b_min(B_real, H, 1, 5, lib=lib)
            b, _ = oracle.allocate(curves, B_real, 1, 5, 40, mode=2, lib=lib)
            assert b.sum() == B_real and (b >= bmin).all()
            _, arg = _brute_force(curves, B_real, bmin)
            assert list(b) == list(arg), (b, arg)
    c = np.array([[10, 6, 4, 3, 2.5, 2.2], [9, 8, 7.5, 3, 2, 1.9]], float)
    b, rep = oracle.allocate(c, 5, 1, 5, 40, mode=2, lib=lib)
    assert b.tolist() == [4, 1] and rep == 3, (b, rep)
    # the safeguard binds: b_min = floor(30 / (5 * 2)) = 3, and head 1 is flat,
    # so greedy keeps it at exactly b_min and gives head 0 the other 27
    c = np.stack([100.0 - np.arange(40.0), np.full(40, 5.0)])
    b, rep = oracle.allocate(c, 30, 1, 5, 40, mode=2, lib=lib)
    assert b.tolist() == [27, 3], b


def _full_attention(q, K, V, scale):
    lg = scale * (K @ q)
    w = np.exp(lg - lg.max())
    return (w[:, None] * V).sum(0) / w.sum()


def _certificate_case(rng, n, d, b, m, spread, scale, lib):
    """A unit with a kept set of b rows and m clusters over the rest; returns
    (O-hat, bound, certified, structural, exact O)."""
    K = to_bf16_bits(rng.normal(size=(n, d)) * spread)
    V = to_bf16_bits(rng.normal(size=(n, d)))
    q = to_bf16_bits(rng.normal(size=d))
    perm = rng.permutation(n).astype(np.int32)
    kb, vb, cnt, rk, rv, _ = oracle.tail_clusters(K, V, perm, b, m, lib=lib)
    kept = perm[:b]
    est, bound, cert, struct = oracle.decode_certified(q, K[kept], V[kept], kb, vb, cnt, rk, rv,
                                                       scale=scale, lib=lib)
    exact = _full_attention(bf(q), bf(K), bf(V), scale)
    return est, bound, cert, struct, exact


def pin_certificate_singleton_clusters_exact(lib=None):
    """Clustered-tail certificate (appendix theorem): with one token per
    cluster every radius is 0 (the stored bf16 representative is the token
    itself), so D_Z = D_N = 0, the bound is 0 and O-hat is exact attention."""
    rng = np.random.default_rng(31)
    n, d, b = 24, 16, 9
    est, bound, cert, struct, exact = _certificate_case(rng, n, d, b, n - b, 1.0, 0.25, lib)
    assert cert and bound == 0.0 and struct == 0.0
    assert np.abs(est - exact).max() < 1e-12


def pin_certificate_bound_holds(lib=None):
    """The runtime bound dominates the true output error whenever its
    checkable condition D_Z <= Z-hat / 3 holds (appendix theorem, Eq.
    (certificate-bound)), and it is at most its structural form (Eq.
    (certificate-structure)); tighter key clusters give smaller bounds."""
    rng = np.random.default_rng(32)
    held = 0
    for trial in range(40):
        n, d = int(rng.integers(20, 60)), int(rng.choice([8, 16, 32]))
        b = int(rng.integers(1, n - 2))
        m = int(rng.integers(1, n - b + 1))
        spread = float(rng.choice([0.02, 0.1, 0.5]))
        est, bound, cert, struct, exact = _certificate_case(rng, n, d, b, m, spread, 0.3, lib)
        if cert:
            held += 1
            assert np.linalg.norm(est - exact) <= bound * (1 + 1e-9) + 1e-12, (trial, bound)
            assert bound <= struct * (1 + 1e-9) + 1e-12, (trial, bound, struct)
    assert held >= 20
    rng = np.random.default_rng(33)
    loose = _certificate_case(rng, 40, 16, 10, 3, 0.5, 0.3, lib)[1]
    rng = np.random.default_rng(33)
    tight = _certificate_case(rng, 40, 16, 10, 3, 0.05, 0.3, lib)[1]
    assert tight < loose


def pin_certificate_value_radius(lib=None):
    """Identical keys inside each cluster make every logit radius 0, so the
    only error left is the value representative (rounded to bf16): it must be
    covered by the value-radius term rho_g of D_N alone."""
    rng = np.random.default_rng(36)
    n, d, b, m = 48, 16, 8, 4
    T = n - b
    perm = rng.permutation(n).astype(np.int32)
    Kf = rng.normal(size=(n, d))
    for g in range(m):  # one key per cluster
        rows = perm[b + g * T // m: b + (g + 1) * T // m]
        Kf[rows] = rng.normal(size=d)
    K, V = to_bf16_bits(Kf), to_bf16_bits(rng.normal(size=(n, d)) * 3.0)
    q = to_bf16_bits(rng.normal(size=d))
    kb, vb, cnt, rk, rv, _ = oracle.tail_clusters(K, V, perm, b, m, lib=lib)
    assert np.allclose(rk, 0.0)
    est, bound, cert, _ = oracle.decode_certified(q, K[perm[:b]], V[perm[:b]], kb, vb, cnt, rk, rv,
                                                  scale=0.25, lib=lib)
    err = np.linalg.norm(est - _full_attention(bf(q), bf(K), bf(V), 0.25))
    assert cert and 0.0 < err <= bound, (err, bound)


def pin_certificate_logit_radius(lib=None):
    """Hand-built case where the logit radius matters: q = (32, 0, 0, 0),
    scale 1/2; one kept token (key e1 / 2, value e1, logit 8) and one tail cluster
    of three keys (2, -1, -1) e1 / 32 (centroid exactly 0, key radius 1/16,
    logits 1, -1/2, -1/2) sharing the value e2 (value radius 0).  The logit
    radius is scale ||q|| 1/16 = 1; the estimator puts weight 3 on e2 where
    exact attention puts e + 2 e^{-1/2} = 3.93 beside e^8 on e1, an output error
    of 4.41e-4, inside the bound 3/Z-hat (D_N + V'max D_Z) = 0.0282 but not
    inside what a radius without the query norm (1/32) would give (1.98e-4)."""
    d = 4
    K = to_bf16_bits(np.array([[0.5, 0, 0, 0], [2 / 32, 0, 0, 0], [-1 / 32, 0, 0, 0],
                               [-1 / 32, 0, 0, 0]], float))
    V = to_bf16_bits(np.array([[1, 0, 0, 0], [0, 1, 0, 0], [0, 1, 0, 0], [0, 1, 0, 0]], float))
    q = to_bf16_bits(np.array([32.0, 0, 0, 0]))
    perm = np.arange(4, dtype=np.int32)
    kb, vb, cnt, rk, rv, _ = oracle.tail_clusters(K, V, perm, 1, 1, lib=lib)
    assert cnt.tolist() == [3] and rk[0] == 1 / 16 and rv[0] == 0.0
    est, bound, cert, _ = oracle.decode_certified(q, K[:1], V[:1], kb, vb, cnt, rk, rv,
                                                  scale=0.5, lib=lib)
    err = np.linalg.norm(est - _full_attention(bf(q), bf(K), bf(V), 0.5))
    assert cert and abs(err - 4.408e-4) < 1e-6 and err <= bound, (err, bound)
    assert abs(bound - 0.02818) < 1e-4, bound


def pin_cluster_summaries(lib=None):
    """Cluster summaries: consecutive rank groups of the evicted tail (reading
    R-C1) with the bf16-rounded unweighted means and the largest distances to
    them as radii (reading R-C2), checked by direct computation."""
    rng = np.random.default_rng(34)
    n, d, b, m = 30, 8, 7, 4
    K = to_bf16_bits(rng.normal(size=(n, d)))
    V = to_bf16_bits(rng.normal(size=(n, d)))
    perm = rng.permutation(n).astype(np.int32)
    kb, vb, cnt, rk, rv, vmax = oracle.tail_clusters(K, V, perm, b, m, lib=lib)
    T = n - b
    assert cnt.tolist() == [(g + 1) * T // m - g * T // m for g in range(m)]
    for g in range(m):
        rows = perm[b + g * T // m: b + (g + 1) * T // m]
        assert (kb[g] == to_bf16_bits(bf(K[rows]).mean(0))).all()
        assert (vb[g] == to_bf16_bits(bf(V[rows]).mean(0))).all()
        assert abs(rk[g] - np.linalg.norm(bf(K[rows]) - bf(kb[g]), axis=1).max()) < 1e-12
        assert abs(rv[g] - np.linalg.norm(bf(V[rows]) - bf(vb[g]), axis=1).max()) < 1e-12
    assert abs(vmax - np.linalg.norm(bf(V[perm[:b]]), axis=1).max()) < 1e-12


def pin_packed_layout_with_clusters(lib=None):
    """With m cluster summaries per head every head is charged m more slots
    (exact-budget accounting): sum_h b_h = B_live - H (tail_slot + m), each
    segment is its b_h real slots, the tail slot, then the m summary slots
    (positions -2 - g), and every (sequence, layer) still fills exactly B_live
    slots."""
    rng = np.random.default_rng(35)
    B, L, Hq, H, n, d, w, m = 1, 2, 4, 2, 64, 8, 4, 3
    K = to_bf16_bits(rng.normal(size=(B, L, H, n, d)))
    V = to_bf16_bits(rng.normal(size=(B, L, H, n, d)))
    Q = to_bf16_bits(rng.normal(size=(B, L, Hq, w, d)))
    B_live = 30
    r = oracle.compress(K, V, Q, B=B, L=L, Hq=Hq, H=H, n=n, d=d, w=w, B_live=B_live,
                        clusters=m, threads=1, lib=lib)
    for bl in range(B * L):
        cnt = r["counts"][bl * H:(bl + 1) * H]
        assert cnt.sum() == B_live - H * (1 + m), cnt
        for h in range(H):
            u = bl * H + h
            off, end = r["offsets"][u], r["offsets"][u + 1]
            assert end - off == cnt[h] + 1 + m
            pos = r["positions"][off:end]
            assert (pos[:cnt[h]] >= 0).all() and pos[cnt[h]] == -1
            assert pos[cnt[h] + 1:].tolist() == [-2 - g for g in range(m)]
            assert int(r["cl_meta"][u, :, 0].sum()) == n - cnt[h]
    assert r["offsets"][-1] == B * L * B_live


def pin_fixed_row_three_tokens(lib=None):
    """Fixed-row quantities in closed form: q = e1, scale 1, keys 0, 0, e1
    (logits 0, 0, 1, so A = (1, 1, e) / (2 + e)), values e1, e2, (1, 1), the
    first token kept: p_S = 1/(2+e), O = (1+e)(1, 1)/(2+e), O~_S = e1,
    u* = (e, 1+e)/(2+e), V_max = sqrt 2."""
    e = math.e
    o = (1 + e) / (2 + e)
    want = [1 / (2 + e), math.sqrt(2) * o, math.hypot(1 - o, o), math.hypot(e / (2 + e), o),
            2 * math.sqrt(2) * (1 - 1 / (2 + e))]
    st = oracle.fixed_row(to_bf16_bits([1.0, 0.0]), to_bf16_bits([[0, 0], [0, 0], [1, 0]]),
                          to_bf16_bits([[1, 0], [0, 1], [1, 1]]), np.array([1, 0, 0]), scale=1.0,
                          lib=lib)
    for i, w in enumerate(want):
        assert abs(st[i] - w) < 1e-12, (i, st[i], w)


def pin_fixed_row_factorization(lib=None):
    """Theorem (fixed-row tail factorization) on random rows: O = p_S O~_S +
    (1 - p_S) V-bar_T exactly (residual at rounding level), the subset-only
    error obeys ||O~_S - O|| <= 2 V_max (1 - p_S), keeping every token gives
    p_S = 1 and no error, and ohat = O gives no error."""
    rng = np.random.default_rng(41)
    for _ in range(20):
        n, d = int(rng.integers(5, 80)), int(rng.choice([4, 16]))
        K = to_bf16_bits(rng.normal(size=(n, d)))
        V = to_bf16_bits(rng.normal(size=(n, d)))
        q = to_bf16_bits(rng.normal(size=d))
        kept = rng.random(n) < 0.3
        kept[0] = True
        st = oracle.fixed_row(q, K, V, kept, scale=0.5, lib=lib)
        assert st[7] < 1e-12 and st[2] <= st[4] * (1 + 1e-12)
        lg = 0.5 * (bf(K) @ bf(q))
        w = np.exp(lg - lg.max())
        exact = (w[:, None] * bf(V)).sum(0) / w.sum()
        st2 = oracle.fixed_row(q, K, V, kept, scale=0.5, ohat=exact, lib=lib)
        assert st2[5] < 1e-12
        st3 = oracle.fixed_row(q, K, V, np.ones(n, bool), scale=0.5, lib=lib)
        assert abs(st3[0] - 1.0) < 1e-15 and st3[2] < 1e-12 and st3[3] < 1e-12


def pin_future_query_lift_worked(lib=None):
    """Theorem (future-query lift) on a hand-built row: q = e1, scale 1, keys
    0, 0, e1 (logits 0, 0, 1), values e1, e2, (1, 1), the first token kept;
    tail weights r = (1/4, 3/4) and the slot (k*, v*) = (e1/2, (3/4, 1)), so
    z* = 1/2 and v* is exactly the r-mixture.  Closed forms: p = (1+e)/(2+e),
    q = sqrt(e)/(1+sqrt(e)), a = (1, e)/(1+e), Lambda_T = log(1+e)."""
    e, se = math.e, math.sqrt(math.e)
    p, qs = (1 + e) / (2 + e), se / (1 + se)
    l1 = abs(1 / (1 + e) - 0.25) + abs(e / (1 + e) - 0.75)
    lam = math.log(1 + e) - 0.5
    lift = (abs(1 / (2 + e) - 1 / (1 + se)) + abs(1 / (2 + e) - qs / 4)
            + abs(e / (2 + e) - 3 * qs / 4))
    want = [p, qs, l1, lam, math.sqrt(2) * (2 * abs(p - qs) + min(p, qs) * l1),
            math.tanh(abs(lam) / 4), lift, 0.0]
    st = oracle.future_query_lift(
        to_bf16_bits([1.0, 0.0]), to_bf16_bits([[0, 0], [0, 0], [1, 0]]),
        to_bf16_bits([[1, 0], [0, 1], [1, 1]]), np.array([1, 0, 0]),
        np.array([0.5, 0.25, 0.75], np.float32), scale=1.0,
        kstar=to_bf16_bits([0.5, 0.0]), vstar=to_bf16_bits([0.75, 1.0]), lib=lib)
    for i, w in enumerate(want):
        assert abs(st[i] - w) < 1e-12, (i, st[i], w)
    # without a slot the compressed row is the kept set alone: q = 0 and
    # ||A - Abar||_1 = 2p, the bound 2 V_max p
    st0 = oracle.future_query_lift(
        to_bf16_bits([1.0, 0.0]), to_bf16_bits([[0, 0], [0, 0], [1, 0]]),
        to_bf16_bits([[1, 0], [0, 1], [1, 1]]), np.array([1, 0, 0]),
        np.array([0.5, 0.25, 0.75], np.float32), scale=1.0, lib=lib)
    assert st0[1] == 0.0 and abs(st0[6] - 2 * p) < 1e-12
    assert abs(st0[4] - 2 * math.sqrt(2) * p) < 1e-12
    assert math.isnan(st0[3]) and math.isnan(st0[5]) and math.isnan(st0[7])


def pin_future_query_lift_single_tail_token(lib=None):
    """With one evicted token t and the slot equal to (k_t, v_t) the compressed
    row is the exact row: p = q, a = r = the point mass, Lambda_T = z*, and
    every mismatch and bound vanishes."""
    rng = np.random.default_rng(43)
    for _ in range(10):
        n, d = int(rng.integers(3, 40)), int(rng.choice([4, 16]))
        K = to_bf16_bits(rng.normal(size=(n, d)))
        V = to_bf16_bits(rng.normal(size=(n, d)))
        q = to_bf16_bits(rng.normal(size=d))
        t = int(rng.integers(n))
        kept = np.ones(n, bool)
        kept[t] = False
        s = rng.random(n).astype(np.float32)
        st = oracle.future_query_lift(q, K, V, kept, s, scale=0.3, kstar=K[t], vstar=V[t],
                                      lib=lib)
        assert abs(st[0] - st[1]) < 1e-15 and 0.0 < st[0] < 1.0
        for i in (2, 3, 4, 5, 6, 7):
            assert abs(st[i]) < 1e-12, (i, st[i])


def pin_future_query_lift_bounds(lib=None):
    """The theorem's inequalities on random rows with a bf16 tail slot built
    from score weights: ||O - Ohat|| <= V_max ||A - Abar||_1 + q ||v* - mixture||
    (Ohat computed here, by plain softmax over S and the slot), ||A - Abar||_1 <=
    2|p - q| + min(p, q) ||a - r||_1, |p - q| <= tanh(|Lambda_T - z*|/4) <=
    |Lambda_T - z*|/4, and p + p_S = 1 with p_S from the fixed-row quantities."""
    rng = np.random.default_rng(47)
    for _ in range(30):
        n, d = int(rng.integers(6, 90)), int(rng.choice([4, 16]))
        K = to_bf16_bits(rng.normal(size=(n, d)) * rng.choice([0.5, 2.0]))
        V = to_bf16_bits(rng.normal(size=(n, d)))
        q = to_bf16_bits(rng.normal(size=d))
        kept = rng.random(n) < 0.4
        kept[0], kept[-1] = True, False
        s = (rng.random(n) ** 3).astype(np.float32)
        Kf, Vf, qf = bf(K), bf(V), bf(q)
        r = np.where(kept, 0.0, s.astype(np.float64))
        r /= r.sum()
        ks, vs = to_bf16_bits(r @ Kf), to_bf16_bits(r @ Vf)
        st = oracle.future_query_lift(q, K, V, kept, s, scale=0.25, kstar=ks, vstar=vs, lib=lib)
        z = 0.25 * (Kf @ qf)
        A = softmax(z)
        O = A @ Vf
        zh = np.concatenate([z[kept], [0.25 * (bf(ks) @ qf)]])
        Ah = softmax(zh)
        Oh = Ah[:-1] @ Vf[kept] + Ah[-1] * bf(vs)
        vmax = np.linalg.norm(Vf, axis=1).max()
        err = np.linalg.norm(O - Oh)
        assert abs(st[1] - Ah[-1]) < 1e-12 and abs(st[0] - A[~kept].sum()) < 1e-12
        assert err <= vmax * st[6] + st[1] * st[7] + 1e-12
        assert st[6] <= 2 * abs(st[0] - st[1]) + min(st[0], st[1]) * st[2] + 1e-12
        assert abs(st[0] - st[1]) <= st[5] + 1e-12 and st[5] <= abs(st[3]) / 4 + 1e-12
        assert st[4] >= vmax * st[6] - 1e-12
        fr = oracle.fixed_row(q, K, V, kept, scale=0.25, lib=lib)
        assert abs(fr[0] + st[0] - 1.0) < 1e-12


def pin_sampled_compensation_worked(lib=None):
    """Sampled tail compensation (appendix proposition) on a hand-built row:
    q = e1, scale 1, logits (2, 0, 0.6875, 0) with token 0 kept, so the tail
    weights are proportional to (1, e^0.6875, 1) and their cumulative shares
    0.2508, 0.7492, 1: uniforms 0.1, 0.3, 0.9 draw tokens 1, 2, 3.  With m = N = 3
    the uniform subset is the whole tail.  Values v0 = 0, v1 = e1, v2 = e2,
    v3 = e1 + e2: u* = (A1 + A3, A2 + A3), Q_T = A1^2 + A2^2 + A3^2."""
    ez = math.exp(0.6875)
    Z = math.e ** 2 + 2 + ez
    A = [math.e ** 2 / Z, 1 / Z, ez / Z, 1 / Z]
    pS, pT = A[0], 1 - A[0]
    K = np.zeros((4, 2)); K[:, 0] = [2.0, 0.0, 0.6875, 0.0]
    V = [[0, 0], [1, 0], [0, 1], [1, 1]]
    kept = np.array([1, 0, 0, 0])
    u = np.array([0.1, 0.3, 0.9, 0.5, 0.5, 0.5], np.float32)
    idx, st = oracle.sampled_compensation(to_bf16_bits([1.0, 0.0]), to_bf16_bits(K),
                                          to_bf16_bits(V), kept, u, scale=1.0, m=3, lib=lib)
    assert idx[:3].tolist() == [1, 2, 3], idx
    assert sorted(idx[3:].tolist()) == [1, 2, 3], idx
    ustar = np.array([A[1] + A[3], A[2] + A[3]])
    uw = pT / 3 * np.array([2.0, 2.0])  # v1 + v2 + v3
    assert abs(st[0] - pS) < 1e-12 and abs(st[1] - (A[1] ** 2 + A[2] ** 2 + A[3] ** 2)) < 1e-12
    assert abs(st[2] - np.linalg.norm(ustar)) < 1e-12
    assert abs(st[3] - np.linalg.norm(uw - ustar)) < 1e-12
    assert abs(st[4] - np.linalg.norm(uw - ustar)) < 1e-12  # the same three tokens
    vbar = np.array([2 / 3, 2 / 3])
    s2 = sum(((np.array(v) - vbar) ** 2).sum() for v in V[1:]) / (2 * 3)
    assert abs(st[7] - s2) < 1e-12


def pin_sampled_compensation_exact_cases(lib=None):
    """A single evicted token is drawn by both samplers and gives u* exactly;
    on a flat row the uniform subset of the whole tail gives u* exactly; with m
    = N the uniform subset holds every tail token once."""
    rng = np.random.default_rng(53)
    for _ in range(6):
        n, d = int(rng.integers(4, 30)), 4
        K = to_bf16_bits(rng.normal(size=(n, d)))
        V = to_bf16_bits(rng.normal(size=(n, d)))
        q = to_bf16_bits(rng.normal(size=d))
        t = int(rng.integers(n))
        kept = np.ones(n, bool); kept[t] = False
        u = rng.random(2).astype(np.float32)
        idx, st = oracle.sampled_compensation(q, K, V, kept, u, scale=0.5, m=1, lib=lib)
        assert idx.tolist() == [t, t] and st[3] < 1e-14 and st[4] < 1e-14
        kept = rng.random(n) < 0.3
        N = int((~kept).sum())
        if N < 2:
            continue
        flat = to_bf16_bits(np.zeros((n, d)))
        u = rng.random(2 * N).astype(np.float32)
        idx, st = oracle.sampled_compensation(q, flat, V, kept, u, scale=0.5, m=N, lib=lib)
        assert sorted(idx[N:].tolist()) == np.flatnonzero(~kept).tolist()
        assert st[4] < 1e-12


def pin_sampled_compensation_mse(lib=None):
    """The proposition's mean-square errors, by Monte Carlo over i.i.d. N(0, 1)
    values and fresh uniforms for one fixed weight row: part (i),
    d (1 - p_S)^2 / m (1 - Q_T/(1 - p_S)^2), and part (ii),
    d (1 - p_S)^2 (1/m - 2/N + Q_T/(1 - p_S)^2), within 8 % (the standard
    error of 6000 trials is ~2 %)."""
    rng = np.random.default_rng(59)
    n, d, m = 24, 4, 3
    K = to_bf16_bits(rng.normal(size=(n, d)))
    q = to_bf16_bits(rng.normal(size=d))
    kept = np.zeros(n, bool); kept[:6] = True
    z = 0.7 * (bf(K) @ bf(q))
    A = np.exp(z - z.max()); A /= A.sum()
    pT = A[~kept].sum(); QT = (A[~kept] ** 2).sum(); N = int((~kept).sum())
    want_w = d * pT ** 2 / m * (1 - QT / pT ** 2)
    want_u = d * pT ** 2 * (1 / m - 2 / N + QT / pT ** 2)
    ew = eu = 0.0
    trials = 6000
    for _ in range(trials):
        V = to_bf16_bits(rng.normal(size=(n, d)))
        u = rng.random(2 * m).astype(np.float32)
        _, st = oracle.sampled_compensation(q, K, V, kept, u, scale=0.7, m=m, lib=lib)
        ew += st[3] ** 2
        eu += st[4] ** 2
    assert abs(ew / trials - want_w) < 0.08 * want_w, (ew / trials, want_w)
    assert abs(eu / trials - want_u) < 0.08 * want_u, (eu / trials, want_u)


def pin_allocation_infeasible(lib=None):
    """B_real above H (n - 1) cannot be met with b_h <= n - 1."""
    curves = np.ones((2, 5))
    try:
        oracle.allocate(curves, 9, lib=lib)
    except ValueError:
        return
    raise AssertionError("infeasible budget accepted")


# --------------------------------------------------------------- tail slot --

def pin_tail_cancellation_witness(lib=None):
    """n = 4, k = 2 witness: top-2 = {1, 2}, truncated error 0.35, and the
    tail correction u* = m v* = -0.35 e2 makes the compensated output exact
    (Theorem 'optimal k-subset', proof step 2; Proposition 'compensation
    exactness')."""
    g = golden("n4_cancellation_witness")
    A = np.array(g["A"])
    V = to_bf16_bits(np.array(g["V"]))
    perm = oracle.order(A, lib=lib)
    kept = oracle.select(perm, g["k"], lib=lib)
    assert kept.tolist() == g["topk_set"]
    ks, vs, m, zero = oracle.tail(A, V, V, perm, g["k"], lib=lib)
    assert not zero
    u = m * vs
    O = np.array(g["O"])
    O_S = (A[kept, None] * bf(V)[kept]).sum(0)
    assert abs(np.linalg.norm(O - O_S) - g["E_topk"]) < 1e-12
    np.testing.assert_allclose(O_S + u, O, atol=1e-12)
    np.testing.assert_allclose(u, -(O_S - O), atol=1e-12)


def pin_tail_factorization(lib=None):
    """Fixed-row tail factorization: with the scorer reduced to one softmax
    row A, O = sum_S A_j v_j + m v* for every kept prefix, where O is the full
    attention output computed independently (Theorem 'fixed-row tail
    factorization'; u* = sum_T A_j V_j = (1 - p_S) bar V_T)."""
    rng = np.random.default_rng(10)
    n, d = 80, 8
    K = to_bf16_bits(rng.standard_normal((n, d)))
    V = to_bf16_bits(rng.standard_normal((n, d)))
    q = to_bf16_bits(rng.standard_normal((1, 1, d)) * 2)
    scale = 1 / math.sqrt(d)
    A = softmax(scale * (bf(K) @ bf(q)[0, 0]))
    O = A @ bf(V)
    a = oracle.scores(K, q, w=1, G=1, scale=scale, pool=1, protect=0, lib=lib)
    perm = oracle.order(a, lib=lib)
    for b in (1, 5, 40, n - 1):
        kept = oracle.select(perm, b, lib=lib)
        ks, vs, m, _ = oracle.tail(a, K, V, perm, b, lib=lib)
        np.testing.assert_allclose(A[kept] @ bf(V)[kept] + m * vs, O, atol=1e-12)
        assert abs(m - (1 - A[kept].sum())) < 1e-12
        # key centroid: same weights on the keys
        np.testing.assert_allclose(m * ks, A[perm[b:]] @ bf(K)[perm[b:]], atol=1e-12)


def pin_flat_row(lib=None):
    """Flat row A_j = 1/n: top-k with ties by index keeps {0..k-1}; with values
    -Vmax e1 kept and +Vmax e1 evicted the truncated error is Vmax (n-k)/n and
    the renormalised error 2 Vmax (n-k)/n (Proposition 'tightness on flat
    rows' (i)); the tail slot makes the output exact."""
    g = golden("flat_row")
    n, k, vm = g["n"], g["k"], g["Vmax"]
    A = np.full(n, 1.0 / n)
    perm = oracle.order(A, lib=lib)
    kept = oracle.select(perm, k, lib=lib)
    assert kept.tolist() == list(range(k))
    V = np.zeros((n, 2))
    V[:, 0] = vm
    V[kept, 0] = -vm
    Vb = to_bf16_bits(V)
    O = A @ V
    O_S = A[kept] @ V[kept]
    assert abs(np.linalg.norm(O_S - O) - vm * (n - k) / n) < 1e-12
    assert abs(np.linalg.norm(O_S / A[kept].sum() - O) - 2 * vm * (n - k) / n) < 1e-12
    ks, vs, m, _ = oracle.tail(A, Vb, Vb, perm, k, lib=lib)
    np.testing.assert_allclose(O_S + m * vs, O, atol=1e-12)


# ----------------------------------------------------------- retained mass --

def _zipf_heads(H=2, n=2048, d=32, w=16, G=4, seed=11):
    """Gaussian keys plus Zipf-weighted planted keys, one recipe per head."""
    rng = np.random.default_rng(seed)
    K = rng.standard_normal((H, n, d))
    Qg = rng.standard_normal((H * G, w, d))
    for h in range(H):
        u = Qg[h * G:(h + 1) * G].reshape(-1, d).mean(0)
        u *= math.sqrt(d) / np.linalg.norm(u)
        pos = rng.choice(n - w, size=32, replace=False)
        for i, p in enumerate(pos):
            K[h, p] = (8.0 if h == 0 else 3.0) * (i + 1) ** -1.1 * u
    V = rng.standard_normal((H, n, d))
    return to_bf16_bits(K), to_bf16_bits(Qg), to_bf16_bits(V)


def pin_retained_mass_bounds(lib=None):
    """On the oracle's scores and allocated top-b_h sets: the order-statistic
    bound 1 - p(k) <= (n-k)/(k+1) (Fact 'order-statistic mass bound'), the
    log-slope envelope 1 - p(k) <= e^b/(gamma-1) k^-(gamma-1) with
    b = max_j (gamma log j - G(j)), G(j) = log(a_(1)/a_(j)), and the n-free
    budget: whenever b_h >= ceil((e^b/((gamma-1) eta))^(1/(gamma-1))) the
    retained mass is at least 1 - eta (Theorem 'coverage regimes from global
    gap envelopes'; Theorem 'log-slope criterion' (i)); plus the plateau
    refinement (Corollary 'plateau sets the sub-linear scale')."""
    H, n, d, w, G = 2, 2048, 32, 16, 4
    K, Qg, V = _zipf_heads(H, n, d, w, G)
    runs = [oracle.compress(K, V, Qg, B=1, L=1, Hq=H * G, H=H, n=n, d=d, w=w,
                            B_live=H * 205, threads=2, lib=lib)]
    # power-law logits l_j = -2.5 log(j + 1) (one observation row, no pooling):
    # a super-logarithmic gap profile, where the n-free budget bound bites
    Kp = np.zeros((H, n, d))
    Kp[0, :, 0] = -2.5 * np.log(np.arange(1, n + 1))
    Kp[1, :, 0] = np.random.default_rng(16).standard_normal(n)
    qp = np.zeros((H, 1, d))
    qp[:, 0, 0] = 1.0
    runs.append(oracle.compress(to_bf16_bits(Kp), V, to_bf16_bits(qp), B=1, L=1, Hq=H, H=H,
                                n=n, d=d, w=1, B_live=H * 205, scale=1.0, pool=1, protect=0,
                                threads=2, lib=lib))
    ks = np.arange(1, n)
    j = np.arange(1, n + 1)
    checked = 0
    for out, h in itertools.product(runs, range(H)):
        a = out["a"][h]
        perm = out["perm"][h]
        srt = a[perm]
        assert (np.diff(srt) <= 0).all()
        p = np.cumsum(srt)
        b_h = int(out["counts"][h])
        assert abs((1 - p[b_h - 1]) - out["tail_mass"][h]) < 1e-12
        assert (1 - p[ks - 1] <= (n - ks) / (ks + 1) + 1e-12).all()
        Gj = np.log(srt[0] / srt)
        for gamma in (1.1, 1.25, 1.5, 2.0, 3.0, 4.0):
            b = max(0.0, float(np.max(gamma * np.log(j) - Gj)))
            bound = math.exp(b) / (gamma - 1) * ks.astype(float) ** (-(gamma - 1))
            assert (1 - p[ks - 1] <= bound * (1 + 1e-12) + 1e-15).all(), gamma
            for eta in (0.5, 0.3, 0.1, 0.01):
                kb = math.ceil((math.exp(b) / ((gamma - 1) * eta)) ** (1 / (gamma - 1)))
                if kb <= b_h:
                    checked += 1
                    assert p[b_h - 1] >= 1 - eta - 1e-12
            J = 16
            b0 = float(Gj[:J].max())
            bj = max(0.0, float(np.max(gamma * np.log(j[J:] / J) - Gj[J:])))
            kk = ks[ks >= J]
            bound = math.exp(bj + b0) / (gamma - 1) * (kk / J) ** (-(gamma - 1))
            assert (1 - p[kk - 1] <= bound * (1 + 1e-12) + 1e-15).all()
    assert checked > 0, "no gap bound applied to the allocated budgets"


def pin_gaussian_kept_fraction(lib=None):
    """iid N(0, 1) logits: K_eta / n is close to Phi(Phi^-1(1 - eta) - 1),
    about 0.61 at eta = 0.1 (§3, 'Count sparsity does not imply coverage
    sparsity').  Uses the scorer's softmax-row special case and the order."""
    g = golden("gaussian_kept_fraction")
    rng = np.random.default_rng(12)
    n = 100_000
    K = np.zeros((n, 2))
    K[:, 0] = rng.standard_normal(n)
    q = np.zeros((1, 1, 2))
    q[0, 0, 0] = 1.0
    a = oracle.scores(to_bf16_bits(K), to_bf16_bits(q), w=1, G=1, scale=g["sigma"], pool=1,
                      protect=0, lib=lib)
    perm = oracle.order(a, lib=lib)
    p = np.cumsum(a[perm])
    k_eta = int(np.searchsorted(p, 1 - g["eta"]) + 1)
    limit = norm.cdf(norm.ppf(1 - g["eta"]) - g["sigma"])
    assert abs(limit - g["value"]) < 0.005
    assert abs(k_eta / n - limit) < 0.01, (k_eta / n, limit)


def pin_coverage_worked(lib=None):
    """Coverage profile of a hand-built row (§3: ranked gap profile G(j) =
    z_(1) - z_(j), coverage budget K_eta, relative and calibrated counts): q =
    e1, scale 1, logits (0, 1, 2, 1/2, 1).  Order 2, 1, 4, 3, 0 (the tied
    logits 1 by lower index), gaps (0, 1, 1, 3/2, 2), Z = e^2 + 2e + sqrt(e) + 1
    (15.474): cumulative ranked mass 0.478, 0.653, 0.829, 0.935, 1, so K_0.5 =
    2, K_0.2 = 3, K_0.05 = 5; A_j > eps A_(1) iff z_j > 2 + log eps (eps 0.3:
    3 tokens, 0.5: 1, 0.1: 5); weights (0.065, 0.176, 0.478, 0.107, 0.176), so
    3 tokens above 0.15 and 4 above 0.1."""
    K = np.zeros((5, 2))
    K[:, 0] = [0.0, 1.0, 2.0, 0.5, 1.0]
    r = oracle.coverage_profile(to_bf16_bits([1.0, 0.0]), to_bf16_bits(K), scale=1.0,
                                eta=[0.5, 0.2, 0.05], rel_eps=[0.3, 0.5, 0.1],
                                abs_eps=[0.15, 0.1], lib=lib)
    assert r["order"].tolist() == [2, 1, 4, 3, 0]
    assert np.allclose(r["gap"], [0.0, 1.0, 1.0, 1.5, 2.0], rtol=0, atol=1e-15)
    assert r["K_eta"].tolist() == [2, 3, 5]
    assert r["rel"].tolist() == [3, 1, 5]
    assert r["abs"].tolist() == [3, 4]
    Z = math.e ** 2 + 2 * math.e + math.sqrt(math.e) + 1
    assert abs(r["top"][0] - 2.0) < 1e-15 and abs(r["top"][1] - math.log(Z)) < 1e-12


def pin_coverage_flat_row(lib=None):
    """A flat row (all logits equal, A_j = 1/n exactly): index order, zero
    gaps, K_eta = ceil((1 - eta) n) with the threshold met exactly at eta =
    1/2 (the definition's >=), every token above eps A_(1) for eps < 1 and none
    at eps = 1, and A_j = 1/8 is not above 1/8."""
    n = 8
    r = oracle.coverage_profile(to_bf16_bits([1.0, 0.0]), to_bf16_bits(np.zeros((n, 2))),
                                scale=1.0, eta=[0.5, 0.1, 0.3], rel_eps=[0.5, 1.0],
                                abs_eps=[0.125, 0.1], lib=lib)
    assert r["order"].tolist() == list(range(n)) and (r["gap"] == 0).all()
    assert r["K_eta"].tolist() == [4, 8, 6]
    assert r["rel"].tolist() == [8, 0] and r["abs"].tolist() == [0, 8]
    assert abs(r["top"][1] - math.log(n)) < 1e-15


def pin_coverage_gaussian_and_envelopes(lib=None):
    """iid N(0, 1) logits: K_eta / n close to Phi(Phi^-1(1 - eta) - 1) (§3);
    the order-statistic mass bound 1 - p(k) <= (n - k)/(k + 1) caps K_eta; and
    on power-law rows the global gap envelopes of Theorem (coverage regimes from
    global gap envelopes) bound K_eta from above (gamma > 1) and below (gamma' <
    1), with b and b' read off the returned gap profile."""
    g = golden("gaussian_kept_fraction")
    rng = np.random.default_rng(19)
    n = 100_000
    K = np.zeros((n, 2))
    K[:, 0] = rng.standard_normal(n)
    r = oracle.coverage_profile(to_bf16_bits([1.0, 0.0]), to_bf16_bits(K), scale=g["sigma"],
                                eta=[g["eta"]], lib=lib)
    limit = norm.cdf(norm.ppf(1 - g["eta"]) - g["sigma"])
    assert abs(r["K_eta"][0] / n - limit) < 0.01, (r["K_eta"][0] / n, limit)
    for n, gamma in ((4000, 2.0), (4000, 1.5), (20000, 0.5), (20000, 0.2)):
        j = np.arange(1, n + 1)
        G = gamma * np.log(j) + rng.random(n) * 0.5
        G[0] = 0.0
        K = np.zeros((n, 2))
        K[rng.permutation(n), 0] = -G
        for eta in (0.1, 0.3):
            r = oracle.coverage_profile(to_bf16_bits([1.0, 0.0]), to_bf16_bits(K), scale=1.0,
                                        eta=[eta], lib=lib)
            gap, k_eta = r["gap"], int(r["K_eta"][0])
            assert k_eta <= math.ceil((n - eta) / (1 + eta))
            if gamma > 1:
                b = max(0.0, float(np.max(gamma * np.log(j) - gap)))
                cap = math.ceil((math.exp(b) / ((gamma - 1) * eta)) ** (1 / (gamma - 1)))
                assert k_eta <= cap, (n, gamma, eta, k_eta, cap)
            else:
                b2 = max(0.0, float(np.max(gap - gamma * np.log(j))))
                floor_ = (1 - eta) * math.exp(-b2) / 2 * n ** (1 - gamma)
                assert k_eta >= floor_, (n, gamma, eta, k_eta, floor_)


def pin_compress_batching(lib=None):
    """The batched pass scores unit (b, l, h) with the observation rows of query
    heads h*G .. h*G+G-1 of the same (b, l) (query head qh reads KV head qh/G)."""
    rng = np.random.default_rng(17)
    B, L, Hq, H, n, d, w = 2, 1, 6, 3, 40, 8, 3
    G = Hq // H
    K = to_bf16_bits(rng.standard_normal((B, L, H, n, d)))
    V = to_bf16_bits(rng.standard_normal((B, L, H, n, d)))
    Q = to_bf16_bits(rng.standard_normal((B, L, Hq, w, d)))
    out = oracle.compress(K, V, Q, B=B, L=L, Hq=Hq, H=H, n=n, d=d, w=w, B_live=H * 10,
                          threads=1, lib=lib)
    for b, l, h in itertools.product(range(B), range(L), range(H)):
        u = (b * L + l) * H + h
        a = oracle.scores(K[b, l, h], Q[b, l, h * G:(h + 1) * G], w=w, G=G,
                          scale=1 / math.sqrt(d), lib=lib)
        np.testing.assert_array_equal(out["a"][u], a)


# ------------------------------------------------------------ packing / bytes

def pin_packed_layout_and_bytes(lib=None):
    """The packed cache holds exactly B_live slots per (sequence, layer) with no
    padding (implementation appendix: persistent bytes are exact), which for
    Llama-3.1-8B at 64K and 10x gives the paper's 8.59 GB -> 0.86 GB
    (Table 'physical-cache')."""
    rng = np.random.default_rng(13)
    B, L, Hq, H, n, d, w = 2, 2, 4, 2, 48, 8, 4
    K = to_bf16_bits(rng.standard_normal((B, L, H, n, d)))
    V = to_bf16_bits(rng.standard_normal((B, L, H, n, d)))
    Q = to_bf16_bits(rng.standard_normal((B, L, Hq, w, d)))
    B_live = H * (n // 4)
    out = oracle.compress(K, V, Q, B=B, L=L, Hq=Hq, H=H, n=n, d=d, w=w, B_live=B_live,
                          threads=2, lib=lib)
    units = B * L * H
    assert out["offsets"][-1] == B * L * B_live
    for bl in range(B * L):
        cnt = out["counts"][bl * H:(bl + 1) * H]
        assert cnt.sum() + H == B_live
        assert out["offsets"][bl * H] == bl * B_live
    Kr = K.reshape(units, n, d)
    Vr = V.reshape(units, n, d)
    for u in range(units):
        o, c = out["offsets"][u], out["counts"][u]
        pos = out["positions"][o:o + c]
        assert (np.diff(pos) > 0).all()
        assert pos.tolist() == oracle.select(out["perm"][u], c, lib=lib).tolist()
        assert (out["pk"][o:o + c] == Kr[u, pos]).all()
        assert (out["pv"][o:o + c] == Vr[u, pos]).all()
        assert out["positions"][o + c] == -1
        tk = [oracle.f64_to_bf16_bits(x, lib=lib) for x in out["tail"][u, 0]]
        assert out["pk"][o + c].tolist() == tk
    gph = golden("physical_cache")
    Lg, Hg, ng, dg = gph["layers"], gph["kv_heads"], gph["n"], gph["d"]
    full = Lg * Hg * ng * 2 * dg * 2
    live = Hg * (ng * gph["keep_num"] // gph["keep_den"])
    packed = Lg * live * 2 * dg * 2
    assert round(full / 1e9, 2) == gph["full_GB"]
    assert round(packed / 1e9, 2) == gph["certkv_GB"]


# -------------------------------------------------------- bf16 rounding ----

def pin_bf16_rounding(lib=None):
    """The tail slot is the centroid rounded once to bf16, to nearest with ties
    to even (reading R-A10).  Pinned against torch's float32 -> bfloat16
    conversion on every value that is exactly a float32 (an independent
    round-to-nearest-even implementation), and on hand-made bit patterns: ties
    at the 8-bit boundary, a value just above a tie that a double -> float32 ->
    bf16 path would round the wrong way, the carry into the exponent, the
    subnormal range and its boundary, the largest finite value and overflow."""
    import torch
    f = lambda x: oracle.f64_to_bf16_bits(x, lib=lib)
    rng = np.random.default_rng(21)
    mant = rng.integers(0, 1 << 23, 4000)
    expo = rng.integers(-149, 128, 4000)
    vals = np.concatenate([
        np.ldexp(1.0 + mant / 2.0 ** 23, expo).astype(np.float32),          # normal and overflow
        (rng.integers(0, 1 << 23, 1000) * 2.0 ** -149).astype(np.float32),  # float32 subnormals
        (rng.standard_normal(2000) * 10.0 ** rng.integers(-30, 30, 2000)).astype(np.float32),
        # exact ties: the low 16 bits of the float32 equal 0x8000
        ((rng.integers(0x00800000, 0x7F000000, 1000) & ~0xFFFF) | 0x8000).astype(np.uint32).view(np.float32),
    ])
    vals = vals[np.isfinite(vals)]
    want = torch.from_numpy(vals.copy()).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = np.array([f(float(x)) for x in vals], np.uint16)
    bad = np.nonzero(got != want)[0]
    assert bad.size == 0, [(float(vals[i]), hex(got[i]), hex(want[i])) for i in bad[:5]]
    cases = [
        (1.0, 0x3F80), (-1.5, 0xBFC0), (0.0, 0x0000), (-0.0, 0x8000),
        (1.0 + 2.0 ** -8, 0x3F80),                  # tie between 0x3F80 (even) and 0x3F81
        (1.0 + 3 * 2.0 ** -8, 0x3F82),              # tie between 0x3F81 and 0x3F82 (even)
        (1.0 + 2.0 ** -8 + 2.0 ** -40, 0x3F81),     # just above a tie: one rounding step
        (1.0 + 2.0 ** -8 - 2.0 ** -40, 0x3F80),     # just below it
        (2.0 - 2.0 ** -8, 0x4000),                  # tie above 0x3FFF: carry into the exponent
        (2.0 - 2.0 ** -9, 0x4000),
        (2.0 - 2.0 ** -7, 0x3FFF),
        (2.0 ** -126, 0x0080),                      # smallest normal
        (2.0 ** -133, 0x0001),                      # smallest subnormal
        (2.0 ** -134, 0x0000),                      # half of it: tie to even (zero)
        (3 * 2.0 ** -134, 0x0002),                  # 1.5 quanta: tie to even (2)
        (2.0 ** -134 + 2.0 ** -160, 0x0001),        # just above half a quantum
        (2.0 ** -126 - 2.0 ** -134, 0x0080),        # tie between 0x007F and the smallest normal
        (127 * 2.0 ** -133, 0x007F),                # largest subnormal
        ((2.0 - 2.0 ** -7) * 2.0 ** 127, 0x7F7F),   # largest finite
        ((2.0 - 2.0 ** -8) * 2.0 ** 127, 0x7F80),   # tie above it: overflow to infinity
        ((2.0 - 2.0 ** -8 - 2.0 ** -30) * 2.0 ** 127, 0x7F7F),
        (-1e39, 0xFF80), (float("inf"), 0x7F80), (float("-inf"), 0xFF80),
    ]
    for x, bits in cases:
        assert f(x) == bits, (x, hex(f(x)), hex(bits))


# ------------------------------------------------------------------ decode --

def pin_decode_textbook(lib=None):
    """Decode over the packed cache is plain softmax attention over each
    segment's slots, the tail slot included (reading R-A12)."""
    rng = np.random.default_rng(14)
    B, L, Hq, H, d = 1, 2, 4, 2, 8
    counts = np.array([3, 5, 2, 4], np.int32)
    offsets = np.concatenate([[0], np.cumsum(counts + 1)]).astype(np.int64)
    slots = int(offsets[-1])
    pk = to_bf16_bits(rng.standard_normal((slots, d)))
    pv = to_bf16_bits(rng.standard_normal((slots, d)))
    q = to_bf16_bits(rng.standard_normal((B, L, Hq, d)))
    out = oracle.decode(q, pk, pv, offsets, counts, B=B, L=L, Hq=Hq, H=H, d=d, lib=lib)
    G = Hq // H
    for bl in range(B * L):
        for qh in range(Hq):
            u = bl * H + qh // G
            seg = slice(offsets[u], offsets[u] + counts[u] + 1)
            p = softmax(bf(pk[seg]) @ bf(q).reshape(-1, Hq, d)[bl, qh] / math.sqrt(d))
            np.testing.assert_allclose(out.reshape(-1, Hq, d)[bl, qh], p @ bf(pv[seg]),
                                       rtol=1e-12, atol=1e-13)


def pin_future_query_lift(lib=None):
    """For fresh decode queries the packed cache obeys the a-posteriori bound
    ||O - O_hat|| <= Vmax (2|p - q| + min(p, q) ||a - r||_1) of Theorem
    'a posteriori future-query lift' (retained logits unchanged), plus the
    bf16 rounding of the stored tail value."""
    rng = np.random.default_rng(15)
    B, L, Hq, H, n, d, w = 1, 1, 2, 1, 64, 8, 4
    K = to_bf16_bits(rng.standard_normal((B, L, H, n, d)))
    V = to_bf16_bits(rng.standard_normal((B, L, H, n, d)))
    Q = to_bf16_bits(rng.standard_normal((B, L, Hq, w, d)))
    out = oracle.compress(K, V, Q, B=B, L=L, Hq=Hq, H=H, n=n, d=d, w=w, B_live=16, threads=1,
                          lib=lib)
    Kf, Vf = bf(K)[0, 0, 0], bf(V)[0, 0, 0]
    b = int(out["counts"][0])
    perm = out["perm"][0]
    S, T = perm[:b], perm[b:]
    r = out["a"][0][T] / out["a"][0][T].sum()
    vstar_exact = out["tail"][0, 1]
    vstar_packed = bf(out["pv"][b])
    vmax = np.sqrt((Vf ** 2).sum(1)).max()
    for _ in range(20):
        qv = to_bf16_bits(rng.standard_normal((1, 1, Hq, d)))
        o_hat = oracle.decode(qv, out["pk"], out["pv"], out["offsets"], out["counts"], B=1,
                              L=1, Hq=Hq, H=H, d=d, lib=lib)[0, 0]
        for qh in range(Hq):
            qq = bf(qv)[0, 0, qh]
            A = softmax(Kf @ qq / math.sqrt(d))
            O = A @ Vf
            pT = A[T].sum()
            zc = np.concatenate([Kf[np.sort(S)] @ qq, [bf(out["pk"][b]) @ qq]]) / math.sqrt(d)
            qstar = softmax(zc)[-1]
            aT = A[T] / pT
            bound = vmax * (2 * abs(pT - qstar) + min(pT, qstar) * np.abs(aT - r).sum())
            slack = qstar * np.linalg.norm(vstar_packed - vstar_exact) + 1e-12
            assert np.linalg.norm(O - o_hat[qh]) <= bound + slack


ALL_PINS = [v for k, v in sorted(globals().items()) if k.startswith("pin_")]
