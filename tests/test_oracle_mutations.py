"""Planted mistakes in the oracle must each fail at least one pin.

Each case edits one line of a copy of the oracle's C source (a dropped term, a
wrong sign, a wrong index, a transposed operand, a wrong tie rule), compiles it
to a temporary library on the CPU, and runs the oracle pin tests against it in a
subprocess.  The pins must fail for every mutant, and pass for the unmodified copy.
"""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "last_oracle.c")

# (name, exact substring in the source, replacement)
MUTANTS = [
    ("gqa_mapping_modulo", "const int g = h / group;\n  const int64_t total_keys",
     "const int g = h % Hkv;\n  const int64_t total_keys"),
    ("query_key_dropped", "for (int p = 0; p < P; ++p) {\n    const int64_t koff",
     "for (int p = 0; p < P - 1; ++p) {\n    const int64_t koff"),
    ("scale_dropped", "a_out[p] = scale * acc;", "a_out[p] = acc;"),
    ("no_visual_normalisation", "s[i] = s[i] / total;\n  }\n  free(row);",
     "s[i] = s[i] / (double)(L * Hq);\n  }\n  free(row);"),
    ("rows_no_visual_normalisation", "s[i] = s[i] / total;\n  }\n  free(a);",
     "s[i] = s[i] / (double)(L * Hq);\n  }\n  free(a);"),
    ("visual_offset_ignored", "s[i] += row[vis_start[b] + i];", "s[i] += row[i];"),
    ("distance_sign", "float dist = 1.0f - c;", "float dist = 1.0f + c;"),
    ("wrong_norm_index", "float c = (dot * r[i]) * r[j];", "float c = (dot * r[i]) * r[i];"),
    ("delta_max_not_min", "delta[i] = fminf(delta[i], dist);", "delta[i] = fmaxf(delta[i], dist);"),
    ("tie_to_highest_index", "if (best < 0 || p > best_p) { best = i; best_p = p; }\n    }\n    j = best;\n    order_out[t] = j;\n    in_s[j] = 1;\n  }\n  free(xf);",
     "if (best < 0 || p >= best_p) { best = i; best_p = p; }\n    }\n    j = best;\n    order_out[t] = j;\n    in_s[j] = 1;\n  }\n  free(xf);"),
    ("dot_tail_dropped", "if (c < n) acc[l] = fmaf(a[c], b[c], acc[l]);",
     "if (c < n - 1) acc[l] = fmaf(a[c], b[c], acc[l]);"),
    ("seed_not_argmax", "  int j = 0;\n  for (int i = 1; i < N; ++i)\n    if (w[i] > w[j]) j = i;\n  order_out[0] = j;\n  in_s[j] = 1;\n  for (int t = 1; t < k; ++t) {\n    /* Eq. 10",
     "  int j = 0;\n  order_out[0] = j;\n  in_s[j] = 1;\n  for (int t = 1; t < k; ++t) {\n    /* Eq. 10"),
    ("order_not_restored", "while (b >= 0 && idx_out[b] > v)", "while (b >= 0 && idx_out[b] < v)"),
    ("budget_floor", "if (q * den < prod) q += 1;", ""),
    ("topk_tie_to_highest_index", "if (best < 0 || w[i] > w[best]) best = i;",
     "if (best < 0 || w[i] >= w[best]) best = i;"),
    ("topk_lowest_scores", "if (best < 0 || w[i] > w[best]) best = i;",
     "if (best < 0 || w[i] < w[best]) best = i;"),
    ("rows_causal_extent_short", "for (int p = 0; p <= pos; ++p) {\n            const int64_t koff",
     "for (int p = 0; p < pos; ++p) {\n            const int64_t koff"),
    ("rows_position_ignored", "const int pos = row_pos[r];",
     "const int pos = cu_seqlens[b + 1] - cu_seqlens[b] - 1;"),
    ("rows_gqa_modulo", "const int g = h / group;\n          const int64_t qoff = (((int64_t)r",
     "const int g = h % Hkv;\n          const int64_t qoff = (((int64_t)r"),
]

PIN_FILES = [os.path.join(ROOT, "tests", "test_oracle_scores.py"),
             os.path.join(ROOT, "tests", "test_oracle_select.py"),
             os.path.join(ROOT, "tests", "test_oracle_topk.py"),
             os.path.join(ROOT, "tests", "test_oracle_rows.py")]


def _run_pins(lib):
    env = dict(os.environ, LAST_ORACLE_LIB=lib)
    return subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                           *PIN_FILES], cwd=ROOT, env=env, capture_output=True, text=True,
                          timeout=300)


def _build(tmp_path, name, text):
    import oracle
    src = tmp_path / f"{name}.c"
    src.write_text(text)
    return oracle.compile_source(str(src), str(tmp_path / f"lib{name}.so"))


def test_unmodified_copy_passes(tmp_path):
    lib = _build(tmp_path, "orig", open(SRC).read())
    r = _run_pins(lib)
    assert r.returncode == 0, r.stdout[-2000:]


@pytest.mark.parametrize("name,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_mutant_fails_a_pin(tmp_path, name, old, new):
    text = open(SRC).read()
    assert text.count(old) == 1, f"mutation site for {name} not unique/found"
    lib = _build(tmp_path, name, text.replace(old, new))
    r = _run_pins(lib)
    assert r.returncode != 0, f"no pin caught mutant {name}"
