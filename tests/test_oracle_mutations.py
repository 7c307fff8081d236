"""The oracle's pins must reject plausible mistakes.

Each case plants one mistake in a copy of the oracle's C source (on the CPU,
in a temporary directory), compiles it, and runs the oracle pin tests against
the broken copy.  The pins pass on the real oracle (the other test files) and
must fail on every mutant here; a mutant that survives means a pin is missing.
"""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "specflash_oracle.c")

MUTANTS = {
    "accept_test_flipped": ("accept = ((double)u[i] * qt < pt);",
                            "accept = ((double)u[i] * qt > pt);"),
    "residual_q_minus_p": ("double diff = p[y] - (double)qj[y];",
                           "double diff = (double)qj[y] - p[y];"),
    "residual_not_normalised": ("const double target = (double)u[k] * mass;",
                                "const double target = (double)u[k];"),
    "final_draw_from_next_row": ("const float *row_j = rows + (size_t)j * V;",
                                 "const float *row_j = rows + (size_t)(j < k ? j + 1 : j) * V;"),
    "final_draw_reuses_test_uniform": ("const double target = (double)u[k] * mass;",
                                       "const double target = (double)u[j] * mass;"),
    "greedy_last_maximum": ("if (logits[x] > logits[best])",
                            "if (logits[x] >= logits[best])"),
    "temperature_ignored": [("double z = (double)logits[x] / tau;",
                             "double z = (double)logits[x];"),
                            ("p[x] = exp((double)logits[x] / tau - zmax);",
                             "p[x] = exp((double)logits[x] - zmax);")],
    "decisions_past_first_rejection": ("            if (j == k) {\n                if (mg)",
                                       "            {\n                if (mg)"),
    "no_causal_mask": ("const int visible = L + i + 1;", "const int visible = T;"),
    "causal_off_by_one": ("const int visible = L + i + 1;", "const int visible = L + i + (i > 0);"),
    "gqa_modulo_mapping": ("const int h_kv = h / group;", "const int h_kv = h % H_kv;"),
    "scale_dropped": ("        s[t] = scale * acc;\n        if (s[t] > smax)\n            smax = s[t];\n    }\n    double z = 0.0;\n    for (int t = 0; t < visible; ++t)",
                      "        s[t] = acc;\n        if (s[t] > smax)\n            smax = s[t];\n    }\n    double z = 0.0;\n    for (int t = 0; t < visible; ++t)"),
    "slot_shifted": ("int slot = t % page_size;", "int slot = (t + 1) % page_size;"),
    "values_read_from_keys": ("        const uint16_t *vrow =\n            v_cache +",
                              "        const uint16_t *vrow =\n            k_cache +"),
    "commit_keeps_accepted_rows_only": ("const int keep = a + 1 < n_q ? a + 1 : n_q;",
                                        "const int keep = a < n_q ? a : n_q;"),
    "commit_forgets_next_rows": ("*next_len = (long long)(T - n_q) + keep + n_q_next;",
                                 "*next_len = (long long)(T - n_q) + keep;"),
    "commit_takes_top_down": ("            row[lp] = free_pages[take++];",
                              "            row[lp] = free_pages[top - 1 - (take++ - (top - taken))];"),
    "commit_pushes_descending": ("        for (long long lp = need; lp < had; ++lp) {\n            free_pages[sp++] = row[lp];",
                                 "        for (long long lp = need; lp < had; ++lp) {\n            free_pages[sp++] = row[had - 1 - (lp - need)];"),
    "commit_page_count_floor": ("*need = (*next_len + page_size - 1) / page_size;",
                                "*need = *next_len / page_size;"),
    "sample_boundary_inclusive": ("            if (tok < 0 && target < cdf)\n                tok = x;",
                                  "            if (tok < 0 && target <= cdf)\n                tok = x;"),
    "sample_temperature_ignored": ("            pr[x] = exp((double)row[x] / tau - m);",
                                   "            pr[x] = exp((double)row[x] - m * tau);"),
    "sample_greedy_last_max": ("        for (int x = 1; x < V; ++x)\n            if (row[x] > row[best])\n                best = x;",
                               "        for (int x = 1; x < V; ++x)\n            if (row[x] >= row[best])\n                best = x;"),
    "sample_unnormalised_probs": ("            pr[x] /= S;", "            pr[x] /= 1.0;"),
    "compress_scaled_scores": ("                s[n] = acc;\n                if (acc > smax)",
                               "                s[n] = acc / sqrt((double)d);\n                if (acc > smax)"),
    "compress_every_frame_reads_frame_zero": ("        const uint16_t *fv = features + (size_t)f * N * d;",
                                              "        const uint16_t *fv = features;"),
    "compress_weights_not_normalised": ("                const double w = s[n] / z;",
                                        "                const double w = s[n] / (double)N;"),
    "compress_negated_exponent": ("                s[n] = exp(s[n] - smax);",
                                  "                s[n] = exp(smax - s[n]);"),
    "compress_values_from_queries": ("                    o[j] += w * oracle_bf16_value(fv[(size_t)n * d + j]);",
                                     "                    o[j] += w * oracle_bf16_value(qc[j]);"),
    "compress_scores_skip_last_column": ("                for (int j = 0; j < d; ++j)\n                    acc +=",
                                         "                for (int j = 0; j < d - 1; ++j)\n                    acc +="),
}


@pytest.fixture(scope="module")
def source():
    with open(SRC) as f:
        return f.read()


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_reject_mutant(name, source, tmp_path):
    edits = MUTANTS[name]
    edits = edits if isinstance(edits, list) else [edits]
    mutated = source
    for find, repl in edits:
        assert mutated.count(find) == 1, f"mutation anchor for {name} not unique"
        mutated = mutated.replace(find, repl)
    c_path = tmp_path / "mutant.c"
    so_path = tmp_path / "libmutant.so"
    c_path.write_text(mutated)
    subprocess.run(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", str(c_path),
                    "-o", str(so_path), "-lm"], check=True)
    env = dict(os.environ, SPECFLASH_ORACLE_LIB=str(so_path))
    proc = subprocess.run(
        [sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
         os.path.join(ROOT, "tests", "test_oracle_attention.py"),
         os.path.join(ROOT, "tests", "test_oracle_accept.py"),
         os.path.join(ROOT, "tests", "test_oracle_kv_commit.py"),
         os.path.join(ROOT, "tests", "test_oracle_sample.py"),
         os.path.join(ROOT, "tests", "test_oracle_compress.py")],
        cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert proc.returncode != 0, f"mutant {name} survived the oracle pins:\n{proc.stdout[-2000:]}"
