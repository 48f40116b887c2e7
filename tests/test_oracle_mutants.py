"""Planted mistakes in copies of the oracle must each fail at least one pin.

Each mutant is a one-line change to a temporary copy of oracle/fdllm_oracle.c (the
committed file is never touched): a dropped or shifted term, a wrong sign or index, a
flipped comparison, a reversed sort.  The copy is compiled with the same gcc flags and the
whole pin set of ``oracle_pins`` runs against it; a mutant that passes every pin would mean
the pins cannot see that class of mistake.
"""
import os
import shutil

import pytest

import oracle
from oracle_pins import ALL_PINS

MUTANTS = {
    "lower_bound_drops_minus_one": ("sum - (double)(n - 1)", "sum - (double)(n)"),
    "upper_bound_uses_strongest": ("Un[n - 1] = 1.0 - c_sorted[n - 1]",
                                   "Un[n - 1] = 1.0 - c_sorted[0]"),
    "score_sign_flipped": ("Gn[n - 1] = Ln[n - 1] - Un[n - 1]",
                           "Gn[n - 1] = Ln[n - 1] + Un[n - 1]"),
    "no_clip_at_zero": ("Ln[n - 1] = l > 0.0 ? l : 0.0", "Ln[n - 1] = l"),
    "margin_not_strict": ("ok[n - 1] = Gn[n - 1] > delta", "ok[n - 1] = Gn[n - 1] >= delta"),
    "delta_not_matched": ("const double delta = 1.0 - param", "const double delta = param"),
    "factor_drops_plus_one": ("(double)(n + 1) * (1.0 - cs[n - 1])",
                              "(double)(n) * (1.0 - cs[n - 1])"),
    "factor_not_strict": ("ok[n - 1] = r < f", "ok[n - 1] = r <= f"),
    "threshold_strict": ("ok[n - 1] = cs[n - 1] >= tau", "ok[n - 1] = cs[n - 1] > tau"),
    "no_progress_fallback": ("if (nstar == 0)\n            nstar = 1;", ""),
    "first_failure_off_by_one": ("out_tokens[at] = tok[at];\n            out_commit[at] = 1;",
                                 "out_tokens[at] = tok[at];\n            out_commit[at] = j > 0 || nstar == 1;"),
    "sort_ascending": ("if (a->c > b->c)\n        return -1;", "if (a->c > b->c)\n        return 1;"),
    "ties_prefer_higher_position": ("return (a->pos > b->pos) - (a->pos < b->pos);",
                                    "return (a->pos < b->pos) - (a->pos > b->pos);"),
    "argmax_last_of_ties": ("if (arg < 0 || x > M)", "if (arg < 0 || x >= M)"),
    "confidence_is_sum": ("*c_out = 1.0 / S;", "*c_out = S / (double)V;"),
    "exp_sign_flipped": ("S += exp(logit_at(logits, dtype, base + v) - M);",
                         "S += exp(M - logit_at(logits, dtype, base + v));"),
    # the same sum in exact arithmetic, but exp(x) overflows for large logits
    "exp_not_rebased": ("S += exp(logit_at(logits, dtype, base + v) - M);",
                        "S += exp(logit_at(logits, dtype, base + v)) * exp(-M);"),
    "bf16_widened_wrong": ("(uint32_t)((const uint16_t *)logits)[i] << 16",
                           "(uint32_t)((const uint16_t *)logits)[i] << 15"),
    "nan_not_flagged": ("if (saw_nan || !isfinite(M))", "if (!isfinite(M))"),
    "fp16_exponent_bias_off": ("ldexp((double)(1024 + frac), e - 25)",
                               "ldexp((double)(1024 + frac), e - 24)"),
    "fp16_subnormals_scaled_wrong": ("ldexp((double)frac, -24)", "ldexp((double)frac, -25)"),
    "robust_no_clipping": ("const double c_low = c_hat - eta_i > 0.0 ? c_hat - eta_i : 0.0;",
                           "const double c_low = c_hat - eta_i;"),
    "robust_eta_added": ("const double c_low = c_hat - eta_i > 0.0 ? c_hat - eta_i : 0.0;",
                         "const double c_low = c_hat + eta_i;"),
    "robust_ranks_by_c_hat": ("cand[m].c = c_low;", "cand[m].c = c_hat;"),
    "robust_eta_ignored": ("const double eta_i = eta_raw > 0.0 ? eta_raw : 0.0;",
                           "const double eta_i = 0.0;"),
    "robust_negative_eta_kept": ("const double eta_i = eta_raw > 0.0 ? eta_raw : 0.0;",
                                 "const double eta_i = eta_raw;"),
    "factor_core_drops_plus_one": ("Fn[n - 1] = (double)(n + 1) * cn - (double)n;",
                                   "Fn[n - 1] = (double)n * cn - (double)n;"),
    "bonus_index_shifted": ("bonus += c_sorted[j - 1] - cn;", "bonus += c_sorted[j] - cn;"),
    "bonus_sign_flipped": ("bonus += c_sorted[j - 1] - cn;", "bonus += cn - c_sorted[j - 1];"),
    # (old, new, occurrence): the robust selector repeats some lines of the plain one
    "robust_no_progress_fallback": ("if (nstar == 0)\n            nstar = 1;", "", 1),
    "robust_margin_not_strict": ("if (Gn[n - 1] > delta)", "if (Gn[n - 1] >= delta)"),
    "robust_delta_not_matched": ("const double delta = 1.0 - param;", "const double delta = param;",
                                 1),
    # the decision margin: each term dropped or mis-measured
    "margin_drops_next_rank": ("if (nstar < m && fabs(q[nstar]) < mg)\n                mg = fabs(q[nstar]);",
                               ""),
    "margin_at_n_star_only_from_rank": ("double mg = fabs(q[nstar - 1]);", "double mg = INFINITY;"),
    "margin_drops_rank_gap": ("if (gap < mg)\n                mg = gap;", ""),
    "margin_ignores_tie_block": ("if (cs[nstar] != v) {", "if (1) {"),
    "margin_tie_block_ignores_above": ("if (a > 1 && cs[a - 2] - v < mg)\n        mg = cs[a - 2] - v;",
                                       ""),
    "margin_tie_block_ignores_below": ("if (b < m && v - cs[b] < mg)\n        mg = v - cs[b];", ""),
    "robust_margin_drops_clip_gap": ("if (clip_gap < mg)\n                mg = clip_gap;", ""),
    "robust_margin_drops_next_rank": (
        "if (nstar < m && fabs(Gn[nstar] - delta) < mg)\n                mg = fabs(Gn[nstar] - delta);",
        ""),
    "robust_margin_drops_rank_gap": ("if (gap < mg)\n                mg = gap;", "", 1),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_planted_mistake_is_caught(name, tmp_path):
    old, new, *occ = MUTANTS[name]
    which = occ[0] if occ else 0
    with open(oracle.SOURCE) as fh:
        src = fh.read()
    assert src.count(old) > which, "mutation anchor not found: %r" % old
    at = -1
    for _ in range(which + 1):
        at = src.index(old, at + 1)
    src = src[:at] + new + src[at + len(old):]
    shutil.copy(oracle.HEADER, tmp_path / os.path.basename(oracle.HEADER))
    mutated = tmp_path / "mutant.c"
    mutated.write_text(src)
    lib = oracle.compile_oracle(str(mutated), str(tmp_path / "libmutant.so"))
    mut = oracle.Oracle(lib)
    failed = []
    for pin in ALL_PINS:
        try:
            pin(mut)
        except (AssertionError, ValueError, IndexError, OverflowError, FloatingPointError):
            failed.append(pin.__name__)
    assert failed, "planted mistake %s passed every pin" % name
