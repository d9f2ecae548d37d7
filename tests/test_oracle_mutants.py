"""Planted mistakes in the oracle must be caught by its pins (CPU only).

Each case copies the oracle's C source into a temporary directory, plants one
plausible slip (tau multiplied instead of divided, the eps/|C| term dropped,
the tie order reversed, the mean not divided by n_g, the ranking sign flipped,
a transposed operand, a leak of entries outside the selected groups, empty
groups allowed into stage 1, prefix weights reversed, of the wrong sign or
missing the newest element, edge-table rows and columns swapped, an edge
feature misread, edge-prefix weights reversed, Philox words swapped or its key
not advanced, one uniform shared by four groups, the policy's eps term dropped
or tau ignored, the Gumbel noise of the wrong sign, empty groups drawn, the
softmax's log-sum-exp missing its shift or shifted by the first candidate
instead of the largest, the eps/|C| term spread over k_entries, padding slots
weighted, the last candidate dropped from the top-k, stage 1 padding with
group 0, stage 2 reading only the first selected group, a coordinate split
that skips a column of the key sums, group sizes not accumulated), or one
in the Python layer that composes the C routines (the sampled lookup ranking
instead of drawing or dropping tau in stage 2, the edge-routed lookup counting
empty groups, the flat scan ignoring tau, the nearest-key assignment
overwriting given ids, the bf16 rounding of a reduced query truncating or
rounding ties away from zero), builds it there and runs ``test_oracle.py`` against
the mutant: at least one pin has to fail.
"""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

MUTANTS = {
    "tau_multiplied": ("cand[i].score / job->tau - m", "cand[i].score * job->tau - m"),
    "eps_term_dropped": ("job->eps / (double)n_cand +", "0.0 +"),
    "tie_order_reversed": ("if (a->id < b->id) return -1;\n  if (a->id > b->id) return 1;",
                           "if (a->id < b->id) return 1;\n  if (a->id > b->id) return -1;"),
    "mean_not_divided": ("sums[(int64_t)g * d + j] / (double)counts[g]", "sums[(int64_t)g * d + j]"),
    "ranking_sign_flipped": ("if (a->score > b->score) return -1;\n  if (a->score < b->score) return 1;",
                             "if (a->score < b->score) return -1;\n  if (a->score > b->score) return 1;"),
    "operand_transposed": ("load_elem(job->entries, job->e_dtype, e * (int64_t)job->d + j)",
                           "load_elem(job->entries, job->e_dtype, j * (int64_t)job->d + (e % job->d))"),
    "restriction_leaks": ("if (!selected[job->gid[e]]) continue;",
                          "if (!selected[job->gid[e]] && e % 7) continue;"),
    "empty_groups_scored": ("if (job->counts[g] == 0) continue;", ""),
    "prefix_weights_reversed": ("exp(-lambda * (double)(p_len - i))", "exp(-lambda * (double)(i - 1))"),
    "prefix_weight_sign_flipped": ("exp(-lambda * (double)(p_len - i))", "exp(lambda * (double)(p_len - i))"),
    "prefix_newest_dropped": ("for (int32_t i = 1; i <= p_len; ++i) {", "for (int32_t i = 1; i < p_len; ++i) {"),
    "edge_from_to_transposed": ("Z + ((int64_t)from * G + g) * F", "Z + ((int64_t)g * G + from) * F"),
    "edge_feature_misread": ("phi += w[f] * (double)z[f];", "phi += w[f] * (double)z[(f + 1) % F];"),
    "edge_weights_reversed": ("const double alpha = exp(-lambda * (double)(p_len - i));\n      for (int32_t g",
                              "const double alpha = exp(-lambda * (double)(i - 1));\n      for (int32_t g"),
    "philox_words_swapped": ("c[1] = n1;\n    c[2] = n2;\n    c[3] = n3;", "c[1] = n3;\n    c[2] = n2;\n    c[3] = n1;"),
    "philox_key_not_advanced": ("k1 += kPhiloxWeyl1;", "k1 += 0;"),
    "uniform_word_fixed": ("out[g & 3] >> 9", "out[0] >> 9"),
    "policy_eps_dropped": ("mu[o] = eps / (double)n + (1.0 - eps)", "mu[o] = (1.0 - eps)"),
    "policy_tau_ignored": ("if (counts[g] > 0) sum += exp(s[g] / tau - m);", "if (counts[g] > 0) sum += exp(s[g] - m);"),
    "gumbel_sign_flipped": ("keys[o] = log_mu - log(-log(u));", "keys[o] = log_mu + log(-log(u));"),
    "policy_empty_groups_drawn": ("      if (counts[g] == 0) {\n        mu[o] = 0.0;", "      if (0) {\n        mu[o] = 0.0;"),
    "lse_shift_dropped": ("lse_b = m + log(sum);", "lse_b = log(sum);"),
    "softmax_shift_not_max": ("if (z > m) m = z;", "if (i == 0) m = z;"),
    "eps_spread_over_k": ("job->eps / (double)n_cand +", "job->eps / (double)job->k_entries +"),
    "entry_pad_weighted": ("job->entry_weight[o] = 0.0;", "job->entry_weight[o] = job->eps / (double)n_cand;"),
    "topk_drops_last_candidate": ("if (j < n_cand) {\n        job->entry_idx[o]",
                                  "if (j + 1 < n_cand) {\n        job->entry_idx[o]"),
    "stage1_pads_with_group_zero": ("job->group_idx[o] = -1;", "job->group_idx[o] = 0;"),
    "stage2_first_group_only": ("for (int32_t j = 0; j < job->k_groups; ++j) {\n      int32_t g = job->groups",
                                "for (int32_t j = 0; j < 1; ++j) {\n      int32_t g = job->groups"),
    "key_columns_split_short": ("(int32_t)((int64_t)d * (t + 1) / nthreads)",
                                "(int32_t)((int64_t)d * (t + 1) / nthreads) - 1"),
    "counts_not_accumulated": ("counts[gid[e]] += 1;", "counts[gid[e]] = 1;"),
    # Slips in the Python layer that composes the C routines.
    "sampled_lookup_ranks_instead_of_drawing": ("__init__.py", "gi, gk = select(keys, counts, k_groups)",
                                                "gi, gk = select(coarse_scores(queries, centroid), counts, k_groups)"),
    "sampled_stage2_tau_dropped": ("__init__.py",
                                   "gi, k_entries, tau, eps, nthreads)\n    out[\"group_idx\"] = gi\n    out[\"group_key\"]",
                                   "gi, k_entries, 1.0, eps, nthreads)\n    out[\"group_idx\"] = gi\n    out[\"group_key\"]"),
    "edge_lookup_counts_every_group": ("__init__.py",
                                       "counts = np.bincount(np.asarray(gid, dtype=np.int64), minlength=n_groups)",
                                       "counts = np.ones(n_groups, dtype=np.int64)"),
    "flat_tau_ignored": ("__init__.py", "np.zeros((b, 1), np.int32), k_entries, tau, eps,",
                         "np.zeros((b, 1), np.int32), k_entries, 1.0, eps,"),
    "assign_overwrites_given_ids": ("__init__.py", "miss = np.flatnonzero(out == -1)", "miss = np.arange(out.size)"),
    "bf16_rounding_truncates": ("__init__.py", "rounded = (u + 0x7FFF + ((u >> 16) & 1)) >> 16",
                                "rounded = u >> 16"),
    "bf16_ties_away_from_zero": ("__init__.py", "rounded = (u + 0x7FFF + ((u >> 16) & 1)) >> 16",
                                 "rounded = (u + 0x8000) >> 16"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_planted_mistake(name, tmp_path):
    spec = MUTANTS[name]
    target, before, after = spec if len(spec) == 3 else ("htam_oracle.c", *spec)
    (tmp_path / "oracle").mkdir()
    (tmp_path / "tests").mkdir()
    for fname in ("htam_oracle.c", "__init__.py"):
        src = open(os.path.join(ROOT, "oracle", fname)).read()
        if fname == target:
            assert before in src, "mutation site moved; update the mutant"
            src = src.replace(before, after)  # every occurrence
        (tmp_path / "oracle" / fname).write_text(src)
    shutil.copy(os.path.join(ROOT, "tests", "test_oracle.py"), tmp_path / "tests" / "test_oracle.py")
    shutil.copytree(os.path.join(ROOT, "tests", "golden"), tmp_path / "tests" / "golden")
    (tmp_path / "pytest.ini").write_text("[pytest]\naddopts = -p no:cacheprovider\n")
    env = dict(os.environ, PYTHONPATH=str(tmp_path))
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "tests/test_oracle.py"],
                       cwd=tmp_path, env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 1, f"mutant {name} survived the pins:\n{r.stdout[-2000:]}"
