"""The oracle's pins catch plausible mistakes.

Each case copies ``oracle/dpo_oracle.c``, plants one mistake in the copy (a
dropped term, a wrong sign or index, swapped operands, a misread passage),
builds it into a temporary library, and runs ``test_oracle_pins.py`` and
``test_oracle_muon.py`` against that build. Every planted mistake must make at least one pin fail. Nothing
here touches the committed oracle or any GPU.
"""
from __future__ import annotations

import os
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

import pytest

from oracle import build as oracle_build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

# (name, text in dpo_oracle.c, replacement)
MUTANTS = [
    ("decay_on_stale_copy", "hp->eps) + wd * xt)",
     "hp->eps) + wd * (stash != NULL ? stash[i] : xt))"),
    ("eps_inside_sqrt", "(sqrt(v_hat) + hp->eps)", "sqrt(v_hat + hp->eps)"),
    ("ef_sign_flipped", "xn = xt - u - lam * (u - u_prev[i]);",
     "xn = xt - u + lam * (u - u_prev[i]);"),
    ("ef_at_first_update", "corr == ORACLE_CORR_EF && t >= 2", "corr == ORACLE_CORR_EF && t >= 1"),
    ("bias_correction_index", "pow(hp->beta1, (double)k)", "pow(hp->beta1, (double)(k + 1))"),
    ("no_bias_correction_m", "const double m_hat = mi / bc1;", "const double m_hat = mi;"),
    ("stash_holds_new_weights", "stash[i] = oracle_round(xt, hp->stash_store);",
     "stash[i] = oracle_round(xn, hp->stash_store);"),
    ("v_from_momentum", "if (rule == ORACLE_RULE_ADAMW) {\n            mi = hp->beta1 * m[i] + (1.0 - hp->beta1) * gi;\n            vi = hp->beta2 * v[i] + (1.0 - hp->beta2) * gi * gi;",
     "if (rule == ORACLE_RULE_ADAMW) {\n            mi = hp->beta1 * m[i] + (1.0 - hp->beta1) * gi;\n            vi = hp->beta2 * v[i] + (1.0 - hp->beta2) * gi * mi;"),
    ("ema_roles_swapped", "if (rule == ORACLE_RULE_ADAMW) {\n            mi = hp->beta1 * m[i] + (1.0 - hp->beta1) * gi;\n            vi = hp->beta2 * v[i] + (1.0 - hp->beta2) * gi * gi;",
     "if (rule == ORACLE_RULE_ADAMW) {\n            mi = (1.0 - hp->beta1) * m[i] + hp->beta1 * gi;\n            vi = hp->beta2 * v[i] + (1.0 - hp->beta2) * gi * gi;"),
    ("ef_stores_displacement", "double hist = u;", "double hist = xt - xn;"),
    ("clip_not_applied", "double gi = clip_scale * g[i];", "double gi = g[i];"),
    ("clip_no_epsilon", "(sqrt(sqnorm) + 1e-6)", "sqrt(sqnorm)"),
    ("bf16_ties_away", "q = nearbyint(q);", "q = round(q);"),
    ("bf16_subnormal_quantum", "if (e < -125)\n        e = -125;", "if (e < -126)\n        e = -126;"),
    ("decay_ignores_mask", "(wd_on == NULL || wd_on[i])", "(1)"),
    ("sapipe_predicts_with_current_update", "oracle_round(xt - u_prev[i], hp->x_store)",
     "oracle_round(xt - u, hp->x_store)"),
    ("sapipe_updated_bias_index", "bc1_next = 1.0 - pow(hp->beta1, (double)(k + 1))",
     "bc1_next = 1.0 - pow(hp->beta1, (double)k)"),
    ("sapipe_updated_decays_old_weights", "wd * oracle_round(xn, hp->x_store)", "wd * xt"),
    ("sapipe_updated_no_second_blend",
     "const double m2 = hp->beta1 * m[i] + (1.0 - hp->beta1) * gi;", "const double m2 = m[i];"),
    ("delay_mask_ignored", "(delay_on == NULL || delay_on[i])", "(1)"),
    ("ef_restart_counts_all_steps", "corr == ORACLE_CORR_EF && t >= 2",
     "corr == ORACLE_CORR_EF && k >= 2"),
    ("nadam_next_mu_index", "pow(0.96, (double)(k + 1) * hp->momentum_decay)",
     "pow(0.96, (double)k * hp->momentum_decay)"),
    ("lion_roles_swapped", "oracle_round(hp->beta2 * m[i] + (1.0 - hp->beta2) * gi, hp->x_store)",
     "oracle_round(hp->beta1 * m[i] + (1.0 - hp->beta1) * gi, hp->x_store)"),
    ("adan_diff_sign", "const double diff = k == 1 ? 0.0 : gi - g_prev[i];",
     "const double diff = k == 1 ? 0.0 : g_prev[i] - gi;"),
    ("adan_no_lookahead", "gi + hp->beta2 * diff", "gi"),
    ("dc_sign", "(xt - stash[i])", "(stash[i] - xt)"),
    # the updated-state prediction of the rules besides AdamW (App. B.1)
    ("nadam_prediction_gradient_weight_at_k", "(1.0 - mu_next) / (1.0 - mu_prod_next) * gi / d2",
     "(1.0 - mu_k) / (1.0 - mu_prod) * gi / d2"),
    ("nadam_prediction_momentum_weight_at_k", "mu_next2 / (1.0 - mu_prod_next2) * nm / d2",
     "mu_next / (1.0 - mu_prod_next) * nm / d2"),
    ("nadam_prediction_bias_at_k", "sqrt(nv / bc2_next)", "sqrt(nv / bc2)"),
    ("nadam_prediction_no_second_blend",
     "const double nm = hp->beta1 * m[i] + (1.0 - hp->beta1) * gi;", "const double nm = m[i];"),
    ("lion_prediction_is_the_current_update", "hist = hp->lr * (s2 + wd * x_next);",
     "hist = u;"),
    ("lion_prediction_roles_swapped",
     "const double c2 = hp->beta1 * m[i] + (1.0 - hp->beta1) * gi;",
     "const double c2 = hp->beta2 * m[i] + (1.0 - hp->beta2) * gi;"),
    ("adan_prediction_difference_not_decayed",
     "const double av = hp->beta2 * v[i] + (1.0 - hp->beta2) * ad;", "const double av = v[i];"),
    ("adan_prediction_momentum_unblended",
     "const double am = hp->beta1 * m[i] + (1.0 - hp->beta1) * gi;", "const double am = m[i];"),
    ("adan_prediction_bias_at_k", "sqrt(an / bc3_next)", "sqrt(an / bc3)"),
    ("prediction_decays_old_weights_other_rules",
     "const double x_next = oracle_round(xn, hp->x_store);", "const double x_next = xt;"),
    # delayed Muon (Alg. 2) and its Newton-Schulz iteration
    ("ns_coefficient_roles", "AA[i] = oracle_round(b * A[i] + c * AA[i], store);",
     "AA[i] = oracle_round(c * A[i] + b * AA[i], store);"),
    ("ns_drops_linear_term", "X[i] = oracle_round(a * X[i] + BX[i], store);",
     "X[i] = oracle_round(BX[i], store);"),
    ("ns_norm_squared", "const double scale = 1.0 / (sqrt(ss) + eps);",
     "const double scale = 1.0 / (ss + eps);"),
    ("ns_bf16_skips_b", "AA[i] = oracle_round(b * A[i] + c * AA[i], store);",
     "AA[i] = b * A[i] + c * AA[i];"),
    ("ns_output_not_transposed_back", "O[j * cols + i] = X[i * w + j];",
     "O[i * rows + j] = X[i * w + j];"),
    ("muon_momentum_roles",
     "hp->momentum * mom[i] + (1.0 - hp->momentum) * (clip_scale * g[i])",
     "(1.0 - hp->momentum) * mom[i] + hp->momentum * (clip_scale * g[i])"),
    ("muon_sapipe_updated_no_second_blend",
     "M2[i] = oracle_round(hp->momentum * mom[i] + (1.0 - hp->momentum) *\n"
     "                                 (clip_scale * g[i]), hp->x_store);",
     "M2[i] = mom[i];"),
    ("muon_sapipe_updated_decays_the_stash",
     "hp->weight_decay * x[i]), hp->x_store);", "hp->weight_decay * stash[i]), hp->x_store);"),
    ("muon_sapipe_updated_keeps_the_real_update", "    if (updated) {", "    if (0) {"),
    ("muon_scale_smaller_dim", "sqrt((double)(rows > cols ? rows : cols))",
     "sqrt((double)(rows < cols ? rows : cols))"),
    ("muon_decay_on_stash", "hp->lr * (s * O[i] + hp->weight_decay * xt)",
     "hp->lr * (s * O[i] + hp->weight_decay * (hp->delay == 1 ? stash[i] : xt))"),
    ("muon_stash_holds_new_weights", "stash[i] = oracle_round(x[i], hp->stash_store);",
     "stash[i] = oracle_round(xn, hp->stash_store);"),
    ("muon_sapipe_predicts_with_current_update",
     "oracle_round(oracle_round(x[i] - u_prev[i], hp->x_store), hp->stash_store)",
     "oracle_round(oracle_round(x[i] - u, hp->x_store), hp->stash_store)"),
    ("muon_ef_at_first_update", "const int ef_now = use_ef && !sapipe && t >= 2;",
     "const int ef_now = use_ef && !sapipe && t >= 1;"),
    ("lion_sign_of_zero_positive", "(c < 0.0 ? -1.0 : 0.0)", "(c < 0.0 ? -1.0 : 1.0)"),
    ("dc_abs_gradient", "hp->dc_lambda * gi * gi * (xt - stash[i])",
     "hp->dc_lambda * fabs(gi) * (xt - stash[i])"),
    ("dc_on_synchronous_tensors", "if (hp->dc_lambda != 0.0 && delayed)",
     "if (hp->dc_lambda != 0.0)"),
    ("sapipe_prediction_rounded_once",
     "stash[i] = oracle_round(oracle_round(xt - u_prev[i], hp->x_store),\n"
     "                                        hp->stash_store);",
     "stash[i] = oracle_round(xt - u_prev[i], hp->stash_store);"),
    ("muon_ef_lambda_ignored", "xt - u - hp->ef_lambda * (u - u_prev[i])",
     "xt - u - (u - u_prev[i])"),
    ("muon_sapipe_prediction_rounded_once",
     "oracle_round(oracle_round(x[i] - u_prev[i], hp->x_store), hp->stash_store)",
     "oracle_round(x[i] - u_prev[i], hp->stash_store)"),
    ("bf16_weights_from_unrounded_update",
     "        x[i] = oracle_round(xn, hp->x_store);\n        if (param != NULL)\n"
     "            param[i] = oracle_round(x[i], hp->param_store);\n    }\n    return 0;\n}",
     "        x[i] = oracle_round(xn, hp->x_store);\n        if (param != NULL)\n"
     "            param[i] = oracle_round(xn, hp->param_store);\n    }\n    return 0;\n}"),
    ("history_not_stored_in_fp32", "            u_prev[i] = oracle_round(hist, hp->x_store);",
     "            u_prev[i] = hist;"),
    ("muon_master_not_stored_in_fp32",
     "        x[i] = oracle_round(xn, hp->x_store);\n        if (param != NULL)\n"
     "            param[i] = oracle_round(x[i], hp->param_store);\n    }\n    if (o_out",
     "        x[i] = xn;\n        if (param != NULL)\n"
     "            param[i] = oracle_round(x[i], hp->param_store);\n    }\n    if (o_out"),
    ("muon_momentum_not_stored_in_fp32",
     "        mom[i] = oracle_round(hp->momentum * mom[i] + (1.0 - hp->momentum) * (clip_scale * g[i]),"
     "\n                              hp->x_store);",
     "        mom[i] = hp->momentum * mom[i] + (1.0 - hp->momentum) * (clip_scale * g[i]);"),
    ("adan_previous_gradient_unclipped", "g_prev[i] = oracle_round(gi, hp->x_store);",
     "g_prev[i] = oracle_round(g[i], hp->x_store);"),
    ("nadam_gradient_term_unclipped", "(1.0 - mu_k) / (1.0 - mu_prod) * gi / d",
     "(1.0 - mu_k) / (1.0 - mu_prod) * g[i] / d"),
    ("lion_blend_unclipped", "const double c = hp->beta1 * m[i] + (1.0 - hp->beta1) * gi;",
     "const double c = hp->beta1 * m[i] + (1.0 - hp->beta1) * g[i];"),
    ("sapipe_updated_blend_unclipped",
     "const double m2 = hp->beta1 * m[i] + (1.0 - hp->beta1) * gi;",
     "const double m2 = hp->beta1 * m[i] + (1.0 - hp->beta1) * g[i];"),
    ("synchronous_tensor_stash_written", "        if (delayed) {\n            if (corr == ORACLE_CORR_EF)",
     "        if (hp->delay == 1) {\n            if (corr == ORACLE_CORR_EF)"),
    ("lion_sign_after_momentum_update",
     "            const double c = hp->beta1 * m[i] + (1.0 - hp->beta1) * gi;\n"
     "            const double sgn = c > 0.0 ? 1.0 : (c < 0.0 ? -1.0 : 0.0);\n"
     "            u = hp->lr * (sgn + wd * xt);\n"
     "            m[i] = oracle_round(hp->beta2 * m[i] + (1.0 - hp->beta2) * gi, hp->x_store);",
     "            m[i] = oracle_round(hp->beta2 * m[i] + (1.0 - hp->beta2) * gi, hp->x_store);\n"
     "            const double c = hp->beta1 * m[i] + (1.0 - hp->beta1) * gi;\n"
     "            const double sgn = c > 0.0 ? 1.0 : (c < 0.0 ? -1.0 : 0.0);\n"
     "            u = hp->lr * (sgn + wd * xt);"),
    ("adan_first_step_per_delayed_phase", "const double diff = k == 1 ? 0.0 : gi - g_prev[i];",
     "const double diff = t == 1 ? 0.0 : gi - g_prev[i];"),
    ("ns_on_the_larger_gram_matrix", "const int tall = rows > cols;",
     "const int tall = rows < cols;"),
    ("quadratic_gradient_unrounded",
     "grad_out[i] = oracle_round(a[i] * d + (noise ? noise[i] : 0.0), store);",
     "grad_out[i] = a[i] * d + (noise ? noise[i] : 0.0);"),
    ("quadratic_noise_dropped",
     "grad_out[i] = oracle_round(a[i] * d + (noise ? noise[i] : 0.0), store);",
     "grad_out[i] = oracle_round(a[i] * d, store);"),
    ("muon_bf16_weights_from_unrounded_update",
     "        x[i] = oracle_round(xn, hp->x_store);\n        if (param != NULL)\n"
     "            param[i] = oracle_round(x[i], hp->param_store);\n    }\n    if (o_out",
     "        x[i] = oracle_round(xn, hp->x_store);\n        if (param != NULL)\n"
     "            param[i] = oracle_round(xn, hp->param_store);\n    }\n    if (o_out"),
    ("adan_n_bias_by_bc2", "const double d = sqrt(ni / bc3) + hp->eps;",
     "const double d = sqrt(ni / bc2) + hp->eps;"),
    ("adan_update_drops_difference",
     "u = hp->lr * ((mi / bc1 + hp->beta2 * vi / bc2) / d + wd * xt);",
     "u = hp->lr * ((mi / bc1) / d + wd * xt);"),
    ("adan_n_of_gradient_only", "const double w = gi + hp->beta2 * diff;",
     "const double w = gi;"),
    ("nadam_product_excludes_current", "    for (int64_t i = 1; i <= k; ++i)\n        mu_prod",
     "    for (int64_t i = 1; i < k; ++i)\n        mu_prod"),
    ("nadam_momentum_term_uses_mu_k", "mu_next / (1.0 - mu_prod_next) * mi / d",
     "mu_k / (1.0 - mu_prod_next) * mi / d"),
    ("lion_decay_not_scaled_by_lr", "u = hp->lr * (sgn + wd * xt);",
     "u = hp->lr * sgn + wd * xt;"),
    ("adamw_decay_not_scaled_by_lr",
     "u = hp->lr * (m_hat / (sqrt(v_hat) + hp->eps) + wd * xt);",
     "u = hp->lr * (m_hat / (sqrt(v_hat) + hp->eps)) + wd * xt;"),
    ("ef_lambda_ignored", "xn = xt - u - lam * (u - u_prev[i]);", "xn = xt - u - (u - u_prev[i]);"),
    ("sapipe_updated_without_decay",
     "                                 wd * oracle_round(xn, hp->x_store));",
     "                                 0.0 * oracle_round(xn, hp->x_store));"),
    ("synchronous_tensor_history_written", "        if (hist_i) {\n            double hist = u;",
     "        if (use_ef) {\n            double hist = u;"),
    ("param_holds_old_weights",
     "            param[i] = oracle_round(x[i], hp->param_store);\n    }\n    return 0;",
     "            param[i] = oracle_round(xt, hp->param_store);\n    }\n    return 0;"),
    ("muon_rms_scale_ignored", "? hp->rms_scale * sqrt((double)(rows > cols ? rows : cols))",
     "? sqrt((double)(rows > cols ? rows : cols))"),
    ("muon_clip_not_applied", "(1.0 - hp->momentum) * (clip_scale * g[i])",
     "(1.0 - hp->momentum) * g[i]"),
    ("muon_decay_not_scaled_by_lr",
     "const double u = hp->lr * (s * O[i] + hp->weight_decay * xt);",
     "const double u = hp->lr * s * O[i] + hp->weight_decay * xt;"),
    ("ns_eps_inside_sqrt", "const double scale = 1.0 / (sqrt(ss) + eps);",
     "const double scale = 1.0 / sqrt(ss + eps);"),
    ("clip_not_clamped_at_one", "    return coef > 1.0 ? 1.0 : coef;", "    return coef;"),
    ("clip_nan_norm_passes", "    return coef > 1.0 ? 1.0 : coef;",
     "    return coef <= 1.0 ? coef : 1.0;"),
    ("sqnorm_drops_last_block", "        for (int64_t b = 0; b < nb; ++b)" + " " * 36 + "\\\n",
     "        for (int64_t b = 0; b < nb - 1; ++b)" + " " * 32 + "\\\n"),
]


def _dc_before_clip():
    """The DC-ASGD compensation applied to the raw gradient, then clipped."""
    src = open(oracle_build.SRC).read()
    i = src.index("        double gi = clip_scale * g[i];\n")
    tail = "gi = gi + hp->dc_lambda * gi * gi * (xt - stash[i]);"
    j = src.index(tail) + len(tail)
    old = src[i:j]
    new = old.replace("double gi = clip_scale * g[i];", "double gi = g[i];") + \
        "\n        gi = clip_scale * gi;"
    return ("dc_compensates_the_raw_gradient", old, new)


MUTANTS.append(_dc_before_clip())


def _build_mutant(tmp_path, name, old, new):
    src = open(oracle_build.SRC).read()
    assert src.count(old) == 1, f"mutation site for {name} not unique"
    path = tmp_path / f"{name}.c"
    path.write_text(src.replace(old, new))
    return oracle_build.build(force=True, src=str(path),
                              out=str(tmp_path / f"lib{name}.so"))


def _run_pins(lib_path):
    env = dict(os.environ, DPO_ORACLE_LIB=lib_path, OMP_NUM_THREADS="1")
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_oracle_pins.py"),
                        os.path.join(ROOT, "tests", "test_oracle_muon.py")],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    return r.returncode, r.stdout[-600:]


def test_every_planted_mistake_fails_a_pin(tmp_path):
    libs = [(name, _build_mutant(tmp_path, name, old, new)) for name, old, new in MUTANTS]
    with ThreadPoolExecutor(max_workers=min(8, os.cpu_count() or 1)) as ex:
        results = list(ex.map(lambda nl: (nl[0],) + _run_pins(nl[1]), libs))
    survivors = [(n, out) for n, rc, out in results if rc == 0]
    assert not survivors, f"mistakes no pin caught: {[n for n, _ in survivors]}"
    # exit code 1 = tests failed (not a collection or usage error)
    assert all(rc == 1 for _, rc, _ in results), results


# Single mistakes in the oracle's Python drivers (oracle/__init__.py and
# oracle/muon.py): the mode switches and Alg. 1's phase counter live there.
PY_MUTANTS = [
    ("__init__.py", "set_delay_keeps_history", "                self.u_prev[:] = 0.0\n",
     "                pass\n"),
    ("__init__.py", "set_delay_no_restash",
     "            self.stash = round_to(self.x, self.stash_store, self.lib)\n", "            pass\n"),
    ("__init__.py", "set_delay_no_phase_reset", "            self.t = 0\n            self.stash_tag",
     "            self.stash_tag"),
    ("__init__.py", "ef_timing_from_global_k", "g.size, self.k, max(self.t, 1)",
     "g.size, self.k, max(self.k, 1)"),
    ("muon.py", "muon_set_delay_keeps_history", "                    u[...] = 0.0\n",
     "                    pass\n"),
    ("muon.py", "muon_set_delay_no_restash",
     "            self.stash = [round_to(x, self.stash_store, self.lib).reshape(x.shape)\n"
     "                          for x in self.x]\n", "            pass\n"),
    ("muon.py", "muon_set_delay_no_phase_reset",
     "                    u[...] = 0.0\n            self.t = 0\n", "                    u[...] = 0.0\n"),
    ("muon.py", "muon_ef_timing_from_global_k", "rows, cols, max(self.t, 1),",
     "rows, cols, max(self.k, 1),"),
    ("muon.py", "muon_sync_matrix_delayed",
     "dly = self.delay if self.delayed is None or self.delayed[i] else 0", "dly = self.delay"),
    ("muon.py", "muon_clip_per_matrix",
     "            sq = sum(float(self.lib.oracle_sqnorm(g.size, _ptr(g))) for g in grads)",
     "            sq = float(self.lib.oracle_sqnorm(grads[0].size, _ptr(grads[0])))"),
    ("muon.py", "muon_decay_mask_ignored",
     "wd = h.weight_decay if self.wd_on is None or self.wd_on[i] else 0.0",
     "wd = h.weight_decay"),
    ("__init__.py", "decay_mask_ignored", "        self.mask = self._tensor_mask(self.wd_on, n)\n",
     "        self.mask = self._tensor_mask(None, n)\n"),
    ("__init__.py", "delay_mask_ignored",
     "        self.delay_mask = self._tensor_mask(self.delayed, n)\n",
     "        self.delay_mask = self._tensor_mask(None, n)\n"),
    ("__init__.py", "supplied_norm_ignored", "        if sq is None:\n            sq = float(",
     "        if True:\n            sq = float("),
    ("__init__.py", "stale_view_ignores_sync_tensors",
     "            return np.where(self.delay_mask == 1, self.stash, latest), self.stash_tag\n",
     "            return self.stash, self.stash_tag\n"),
    ("__init__.py", "stale_view_in_synchronous_training",
     "        if which == \"stale\" and self.delay == 1:\n",
     "        if which == \"stale\":\n"),
    ("muon.py", "muon_supplied_norm_ignored", "        if sq is None:\n            sq = sum(",
     "        if True:\n            sq = sum("),
    ("__init__.py", "initial_weights_not_rounded",
     "        self.x = round_to(flat, self.x_store, self.lib)\n", "        self.x = flat.copy()\n"),
    ("__init__.py", "initial_param_not_rounded",
     "        self.param = (round_to(self.x, self.param_store, self.lib)\n",
     "        self.param = (self.x.copy()\n"),
    ("muon.py", "muon_initial_weights_not_rounded",
     "        self.x = [round_to(_f64(t), self.x_store, self.lib).reshape(s)\n",
     "        self.x = [_f64(t).copy().reshape(s)\n"),
    ("__init__.py", "fp32_settings_keep_lr", "        return HParams(r(self.lr), r(self.beta1)",
     "        return HParams(self.lr, r(self.beta1)"),
    ("muon.py", "muon_fp32_settings_keep_lr", "        return MuonHParams(r(self.lr), r(self.momentum)",
     "        return MuonHParams(self.lr, r(self.momentum)"),
    ("__init__.py", "stash_tag_not_advanced",
     "        if self.delay == 1:\n            self.stash_tag = self.latest_tag\n        self.latest_tag += 1\n",
     "        self.latest_tag += 1\n"),
]


def _run_py_mutant(root, fname, old, new):
    """The pins against a copy of the oracle package with one driver line
    changed (the copy's tests directory puts the copy first on the path)."""
    import shutil
    shutil.copytree(os.path.join(ROOT, "oracle"), os.path.join(root, "oracle"),
                    ignore=shutil.ignore_patterns("__pycache__"))
    os.makedirs(os.path.join(root, "tests"))
    for f in ("conftest.py", "test_oracle_pins.py", "test_oracle_muon.py"):
        shutil.copy(os.path.join(ROOT, "tests", f), os.path.join(root, "tests", f))
    path = os.path.join(root, "oracle", fname)
    src = open(path).read()
    assert src.count(old) == 1, f"mutation site in {fname} not unique"
    open(path, "w").write(src.replace(old, new))
    env = dict(os.environ, OMP_NUM_THREADS="1")
    env.pop("DPO_ORACLE_LIB", None)
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        "tests/test_oracle_pins.py", "tests/test_oracle_muon.py"],
                       cwd=root, env=env, capture_output=True, text=True, timeout=600)
    return r.returncode


def test_every_planted_driver_mistake_fails_a_pin(tmp_path):
    jobs = [(str(tmp_path / name), f, old, new) for f, name, old, new in PY_MUTANTS]
    with ThreadPoolExecutor(max_workers=min(8, os.cpu_count() or 1)) as ex:
        rcs = list(ex.map(lambda j: _run_py_mutant(*j), jobs))
    survivors = [m[1] for m, rc in zip(PY_MUTANTS, rcs) if rc == 0]
    assert not survivors, f"driver mistakes no pin caught: {survivors}"
    assert all(rc == 1 for rc in rcs), rcs
    # the harness itself: an unchanged copy passes
    assert _run_py_mutant(str(tmp_path / "identity"), "__init__.py",
                          "class DelayedOptimizer:", "class DelayedOptimizer:") == 0


def test_unmutated_copy_passes(tmp_path):
    lib = _build_mutant(tmp_path, "identity", "int oracle_step(", "int oracle_step(")
    rc, out = _run_pins(lib)
    assert rc == 0, out
