"""Plant a plausible mistake in a copy of oracle.c and require that the pin
suite catches it.  This shows that the pins constrain every part of the
oracle: a dropped term, a wrong sign or index, a swapped operand, a
non-strict comparison.  CPU only; the planted copies live in a temp dir."""
import pytest

import oracle
from oracle_pins import ALL_CHECKS

MUTANTS = [
    ("no_max_shift", "s += exp(logit_at(base, dtype, ld, r, j) - m);\n  return m + log(s);",
     "s += exp(logit_at(base, dtype, ld, r, j));\n  return log(s);"),
    ("lse_drops_max", "return m + log(s);", "return log(s);"),
    ("d_sign", "jb->d[r] = ps - pt;", "jb->d[r] = pt - ps;"),
    ("teacher_uses_student_lse", "pt = xt - lt;", "pt = xt - ls;"),
    ("gather_off_by_one", "xs = jb->S ? logit_at(jb->S, jb->dtype, jb->ld, r, y) : NAN;",
     "xs = jb->S ? logit_at(jb->S, jb->dtype, jb->ld, r, (y + 1) % jb->V) : NAN;"),
    ("teacher_gather_uses_student", "xt = logit_at(jb->T, jb->dtype, jb->ld, r, y);",
     "xt = jb->S ? logit_at(jb->S, jb->dtype, jb->ld, r, y) : 0.0;"),
    ("bf16_shift", "((uint32_t)h) << 16", "((uint32_t)h) << 15"),
    ("max_skips_last", "for (int64_t j = 0; j < V; ++j) {\n    double x = logit_at(base, dtype, ld, r, j);\n    if (x > m) m = x;",
     "for (int64_t j = 0; j + 1 < V; ++j) {\n    double x = logit_at(base, dtype, ld, r, j);\n    if (x > m) m = x;"),
    ("sum_skips_first", "for (int64_t j = 0; j < V; ++j) s += exp(",
     "for (int64_t j = 1; j < V; ++j) s += exp("),
    ("turn_mean_wrong_n", "double mean = s_t / (double)n; /* Eq. 4 */", "double mean = s_t / (double)(n + 1);"),
    ("turn_stop_non_strict", "if (st_turn < 0 && cum < lambda[i]) {", "if (st_turn < 0 && cum <= lambda[i]) {"),
    ("token_stop_non_strict", "if (st_row < 0 && cum < lambda[i]) {", "if (st_row < 0 && cum <= lambda[i]) {"),
    ("stop_row_first_of_turn", "st_row = (b - 1) - traj_row_off[i];", "st_row = a - traj_row_off[i];"),
    ("carry_ignored", "double cum = cum_in ? cum_in[i] : 0.0;", "double cum = 0.0;"),
    ("turn_cum_adds_sum", "cum += mean; /* Eq. 5 left-hand side, over new turns only */",
     "cum += s_t;"),
    ("step_turn_adds_sum", "s->cum += mean; /* Eq. 5 */", "s->cum += s->turn_sum_t;"),
    ("step_scores_stopped", "if (s->stopped) {", "if (0) {"),
    ("step_stop_row_next", "int64_t pos = s->rows_seen;", "int64_t pos = s->rows_seen + 1;"),
    ("select_tie_highest", "if (l[k] < l[best]) best = k;", "if (l[k] <= l[best]) best = k;"),
    ("select_gate_non_strict", "(l[K] > alpha)) ++K;", "(l[K] >= alpha)) ++K;"),
    ("select_ignores_mask", "(m == NULL || m[K] != 0) &&", "1 &&"),
    ("select_kmax_all_turns", "while (K < nt && (m == NULL || m[K] != 0) && (l[K] > alpha)) ++K;",
     "for (int32_t q = 0; q < nt; ++q) if ((m == NULL || m[q] != 0) && (l[q] > alpha)) ++K;"),
    ("select_argmax", "if (l[k] < l[best]) best = k;", "if (l[k] > l[best]) best = k;"),
    ("loss_sign", "double term = logp_s ? logp_s[r - base] * dd : 0.0;", "double term = logp_s ? -logp_s[r - base] * dd : 0.0;"),
    ("loss_uses_teacher", "double term = logp_s ? logp_s[r - base] * dd : 0.0;", "double term = logp_s ? lt * dd : 0.0;"),
    ("loss_all_turns_retained", "int turn_retained = (st_turn < 0);", "int turn_retained = 1;"),
    ("loss_first_turn_tested_against_start", "int turn_retained = (st_turn < 0);",
     "int turn_retained = (st_turn < 0) && cum >= lambda[i];"),
    ("loss_first_token_tested_against_start", "if (st_row < 0) {\n            loss += term;",
     "if (st_row < 0 && cum >= lambda[i]) {\n            loss += term;"),
    ("loss_drops_trigger_token", "if (st_row < 0) {\n            loss += term;",
     "if (st_row < 0 && cum + lt >= lambda[i]) {\n            loss += term;"),
    ("profile_wrong_decile", "int64_t j = (10 * (r - a)) / n;", "int64_t j = (10 * (r - a)) / (n + 1);"),
    ("step_loss_teacher", "s->loss += ps * dd;", "s->loss += pt * dd;"),
    ("record_drops_prefix", "int32_t len = keep;", "int32_t len = 0;"),
    ("record_no_clamp", "if (keep > n_turns[x]) keep = n_turns[x];", "if (keep > T_max) keep = T_max;"),
    ("record_prefix_off_by_one", "int32_t keep = k0 ? k0[i] : 0;", "int32_t keep = k0 ? k0[i] + 1 : 0;"),
    ("f32_logit_ignores_row", "    return (double)p[r * ld + j];", "    return (double)p[j];"),
    ("thread_split_drops_row", "jb->r1 = rows * (i + 1) / nthreads;",
     "jb->r1 = rows * (i + 1) / nthreads - (i + 1 < nthreads ? 1 : 0);"),
]


def test_mutant_table_applies():
    src = oracle.SRC.read_text()
    for name, old, new in MUTANTS:
        assert src.count(old) >= 1, f"mutant {name}: pattern not found in oracle.c"


@pytest.mark.parametrize("name,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_pins_catch_mutant(tmp_path, name, old, new):
    src = oracle.SRC.read_text()
    mut = src.replace(old, new)
    assert mut != src
    c = tmp_path / f"oracle_{name}.c"
    c.write_text(mut)
    lib = oracle.OracleLib(oracle.build(force=True, src=c, out=tmp_path / f"lib_{name}.so"))
    failed = []
    for check in ALL_CHECKS:
        try:
            check(lib)
        except (AssertionError, ValueError):
            failed.append(check.__name__)
    assert failed, f"no pin caught the planted mistake {name}"
