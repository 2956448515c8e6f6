"""Plant one mistake at a time in a copy of the oracle (on the CPU) and check
that at least one pin catches it, so that the pins constrain every step."""
import pytest

import oracle
import pins

POOL_OK = """    double acc = 0.0;
    for (int i = j - half; i <= j + half; ++i)
      if (i >= 0 && i < nw) acc += s[i];
    st[j] = acc / (double)pool;"""
POOL_BAD = """    double acc = 0.0; int cnt = 0;
    for (int i = j - half; i <= j + half; ++i)
      if (i >= 0 && i < nw) { acc += s[i]; ++cnt; }
    st[j] = acc / (double)cnt;"""

MUTANTS = {
    "centred_term_dropped": ("const double c2 = m * Q - ww;", "const double c2 = m * Q;"),
    "centred_term_sign": ("const double c2 = m * Q - ww;", "const double c2 = m * Q + ww;"),
    "ties_by_higher_index": ("return (p->j < q->j) ? -1 : (p->j > q->j);",
                             "return (p->j > q->j) ? -1 : (p->j < q->j);"),
    "ascending_order": ("if (p->a > q->a) return -1;\n  if (p->a < q->a) return 1;",
                        "if (p->a > q->a) return 1;\n  if (p->a < q->a) return -1;"),
    "pool_divides_by_count": (POOL_OK, POOL_BAD),
    "no_causal_mask": ("const int visible = nw + t + 1;", "const int visible = n;"),
    "causal_mask_off_by_one": ("const int visible = nw + t + 1;",
                               "const int visible = nw + t;"),
    "window_not_protected": ("st[j] = protect ? smax : s[j];", "st[j] = s[j];"),
    "tail_not_normalised": ("for (int i = 0; i < d; ++i) { kstar[i] /= m; vstar[i] /= m; }",
                            ""),
    "tail_includes_last_kept": ("for (int r = b; r < n; ++r) {\n    const int j = perm[r];\n"
                                "    m += a[j];",
                                "for (int r = (b > 0 ? b - 1 : b); r < n; ++r) {\n"
                                "    const int j = perm[r];\n    m += a[j];"),
    "repair_largest_marginal": ("if (best_h < 0 || delta < best) { best = delta; best_h = h; }",
                                "if (best_h < 0 || delta > best) { best = delta; best_h = h; }"),
    "uniform_remainder_to_high_heads": ("(h < B_real % H ? 1 : 0)", "(h >= H - B_real % H ? 1 : 0)"),
    "greedy_ignores_safeguard": ("for (int h = 0; h < H; ++h) b[h] = lo_b;",
                                 "for (int h = 0; h < H; ++h) b[h] = 1;"),
    "certificate_radius_without_query_norm": ("const double r = scale * qn * rk[g];",
                                              "const double r = scale * rk[g];"),
    "certificate_drops_value_radius": ("DN += er * zg * ((er - 1.0) * vn + rv[g]);",
                                       "DN += er * zg * ((er - 1.0) * vn);"),
    "cluster_groups_overlap_kept": ("const int r0 = b + (int)(((int64_t)g * T) / m),",
                                    "const int r0 = (g == 0 ? b - 1 : b) + (int)(((int64_t)g * T) / m),"),
    "fixed_row_subset_not_renormalised": ("const double os = ZS > 0.0 ? OS[i] / ZS : 0.0;",
                                          "const double os = OS[i] / Z;"),
    "lift_slot_weight_over_all_tokens": ("    if (kept[j]) Zhat += exp(z[j] - c);",
                                         "    Zhat += exp(z[j] - c);"),
    "lift_tail_partition_over_all": ("if (!kept[j]) sumT += exp(z[j] - zmaxT);",
                                     "sumT += exp(z[j] - zmaxT);"),
    "lift_tail_weights_not_renormalised": ("const double a = p > 0.0 ? A / p : 0.0;",
                                           "const double a = A;"),
    "coverage_strict_threshold": ("if (c >= 1.0 - eta[e])", "if (c > 1.0 - eta[e])"),
    "coverage_gap_sign": ("if (gap) gap[r] = z1 - t[r].a;", "if (gap) gap[r] = t[r].a - z1;"),
    "coverage_relative_count_absolute": ("> rel_eps[e] * A1", "> rel_eps[e]"),
    "coverage_calibrated_count_unnormalised": ("if (exp(t[r].a - z1) / Z > abs_eps[e])",
                                               "if (exp(t[r].a - z1) > abs_eps[e])"),
    "sampled_draws_ignore_weights": ("      c += w[tail[t]];", "      c += pT / N;"),
    "sampled_estimate_without_tail_mass": ("    uw[i] *= (1.0 - pS) / m;", "    uw[i] *= 1.0 / m;"),
    "sampled_subset_repeats": ("    idx[m + s] = taken ? tail[i] : tail[t];", "    idx[m + s] = tail[t];"),
    "sampled_qt_is_mass": ("      QT += w[j] * w[j];", "      QT += w[j];"),
    "bisection_inverted": ("if (total > B_real) lam_lo = lam; else lam_hi = lam;",
                           "if (total > B_real) lam_hi = lam; else lam_lo = lam;"),
    "kept_not_sorted": ("qsort(kept, (size_t)b, sizeof(int32_t), cmp_int32);", ""),
    "bf16_truncates": ("double r = nearbyint(ldexp(f, 8));", "double r = floor(ldexp(f, 8));"),
    "bf16_ties_away_from_zero": ("double r = nearbyint(ldexp(f, 8));",
                                 "double r = round(ldexp(f, 8));"),
    "bf16_subnormals_truncate": ("double r = nearbyint(ldexp(ax, 133));",
                                 "double r = floor(ldexp(ax, 133));"),
    "bf16_no_exponent_carry": ("if (r == 256.0) { r = 128.0; e += 1; }", ""),
    "decode_drops_tail_slot": ("const int slots = counts[u] + (tail_slot ? 1 : 0);",
                               "const int slots = counts[u];"),
    "wrong_query_group": ("((size_t)bl * g->Hq + (size_t)h * G) * g->w * d",
                          "((size_t)bl * g->Hq + (size_t)h) * g->w * d"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_planted_mistake_is_caught(name, tmp_path):
    old, new = MUTANTS[name]
    src = oracle.source_text()
    assert src.count(old) >= 1, f"mutation site for {name} not found"
    lib = oracle.load_variant(oracle.compile_variant(src.replace(old, new, 1), str(tmp_path)))
    for pin in pins.ALL_PINS:
        try:
            pin(lib=lib)
        except (AssertionError, ValueError):
            return  # caught
    pytest.fail(f"no pin caught the planted mistake {name!r}")
