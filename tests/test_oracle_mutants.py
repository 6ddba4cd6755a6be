"""The oracle's pins catch plausible mistakes in it.

Each case plants one mistake in a copy of ``oracle/kvec_oracle.c`` (a dropped
term, a wrong sign, an off-by-one index, a swapped operand, a wrong reduction),
builds the copy with the oracle's own compiler flags, and runs the pins
(``test_oracle_pins.py``, ``test_golden.py``) against it in a child process:
every planted mistake must fail at least one of them.  The mistakes sit in the
steps of Algorithm 1 and Sections 4.1-4.2 that the pins are meant to hold:
the causal softmax of the window rows, Eq. 1's observation windows, the group
sum, the head-max importance, pooling, sigma and the choice of the delta
extended-window heads, the preserve rule, the coverage-adjusted score P', the
window tail, the update of n_t, and the head-wise adaptive fill.  Runs on the
CPU only.
"""
import os
import shutil
import subprocess
import sys

import pytest

import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "kvec_oracle.c")
HDR = os.path.join(ROOT, "oracle", "kvec_oracle.h")

# (name, text in kvec_oracle.c, its planted replacement); each text occurs once.
MUTANTS = [
    ("causal_mask_one_key_short",
     "const int pos = L - w + q;",
     "const int pos = L - w + q - 1;"),
    ("obs_window_one_row_early",
     "for (int q = w - O; q < w; ++q)\n                for (int t = 0; t < L; ++t) PO[",
     "for (int q = w - O - 1; q < w - 1; ++q)\n                for (int t = 0; t < L; ++t) PO["),
    ("ext_window_uses_O",
     "for (int q = w - Oe; q < w; ++q)",
     "for (int q = w - O; q < w; ++q)"),
    ("group_sum_drops_last_query_head",
     "for (int j = 0; j < g; ++j)\n                for (int q = 0; q < w; ++q) {",
     "for (int j = 0; j < g - 1; ++j)\n                for (int q = 0; q < w; ++q) {"),
    ("importance_sums_heads_instead_of_max",
     "if (x > m) m = x;",
     "m += x;"),
    ("max_pool_drops_right_neighbour",
     "for (int j = lo + 1; j <= hi; ++j) if (x[j] > m) m = x[j];",
     "for (int j = lo + 1; j < hi; ++j) if (x[j] > m) m = x[j];"),
    ("sigma_population_std",
     "sigma[h] = sqrt(ss / (Lc - 1));",
     "sigma[h] = sqrt(ss / Lc);"),
    ("extended_window_for_highest_sigma",
     "if (sigma[o] < sigma[h] || (sigma[o] == sigma[h] && o < h)) ++rank;",
     "if (sigma[o] > sigma[h] || (sigma[o] == sigma[h] && o < h)) ++rank;"),
    ("extended_and_plain_scores_swapped",
     "htop[h] ? PpOe[(size_t)h * Lc + t] : PpO[(size_t)h * Lc + t];",
     "htop[h] ? PpO[(size_t)h * Lc + t] : PpOe[(size_t)h * Lc + t];"),
    ("preserve_count_rounds_up",
     "int k = (int)floor(p->beta * (double)budget);",
     "int k = (int)ceil(p->beta * (double)budget);"),
    ("coverage_sign_flipped",
     "double focus = Ip[t] * (1.0 - coverage);",
     "double focus = Ip[t] * (1.0 + coverage);"),
    ("coverage_layer_count_off_by_one",
     "(double)n_t[t] / ((double)layers_done + 1.0);",
     "(double)n_t[t] / ((double)layers_done + 2.0);"),
    ("lambda_term_dropped",
     "pph[t] = Ph[t] + p->lambda * focus;",
     "pph[t] = Ph[t];"),
    ("preserved_tokens_not_kept",
     "for (int t = 0; t < Lc; ++t) if (ph[t]) kh[t] = 1;",
     ""),
    ("window_tail_not_kept",
     "for (int t = Lc; t < L; ++t) kh[t] = 1;",
     ""),
    ("coverage_counts_head_zero_only",
     "for (int h = 0; h < Hkv; ++h) any |= keep[(size_t)h * L + t];",
     "for (int h = 0; h < 1; ++h) any |= keep[(size_t)h * L + t];"),
    ("adaptive_own_share_rounds_up",
     "*f0 = p->head_budget ? (int)floor(p->ada_floor * (double)*F) : *F;",
     "*f0 = p->head_budget ? (int)ceil(p->ada_floor * (double)*F) : *F;"),
    ("adaptive_joint_fill_one_short",
     "top_k(jk, ja, (int)n, Hkv * (k2 - f0), js);",
     "top_k(jk, ja, (int)n, Hkv * (k2 - f0) - 1, js);"),
    ("adaptive_joint_ranks_plain_scores",
     "jk[i] = Pp[i];",
     "jk[i] = P[i];"),
]


@pytest.fixture(scope="module")
def _gcc():
    if shutil.which("gcc") is None:
        pytest.skip("needs gcc")


def test_every_planted_text_occurs_once():
    src = open(SRC).read()
    for name, old, new in MUTANTS:
        assert src.count(old) == 1, f"{name}: the planted text must occur exactly once"
        assert old != new


def _run_pins_on(tmp_path, text):
    """Builds `text` as the oracle and runs the pins on it in a child process."""
    mutant = tmp_path / "kvec_oracle.c"
    mutant.write_text(text)
    shutil.copy(HDR, tmp_path / "kvec_oracle.h")
    lib = tmp_path / "libkvec_oracle_copy.so"
    oracle.compile_source(str(mutant), str(lib))
    env = dict(os.environ, KVEC_ORACLE_LIB=str(lib), OMP_NUM_THREADS="4")
    return subprocess.run(
        [sys.executable, "-m", "pytest", "-x", "-q", "-m", "not gpu", "-p", "no:cacheprovider",
         os.path.join(ROOT, "tests", "test_oracle_pins.py"), os.path.join(ROOT, "tests", "test_golden.py")],
        cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)


def test_unmodified_copy_passes_the_pins(_gcc, tmp_path):
    r = _run_pins_on(tmp_path, open(SRC).read())
    assert r.returncode == 0, f"{r.stdout[-3000:]}\n{r.stderr[-2000:]}"


@pytest.mark.parametrize("name,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_pins_catch_planted_mistake(_gcc, tmp_path, name, old, new):
    src = open(SRC).read()
    assert src.count(old) == 1
    r = _run_pins_on(tmp_path, src.replace(old, new))
    # 1: some pin failed (0 would mean the mistake went unnoticed; 2-5 are pytest's
    # own errors, which would not show that a pin holds the step).
    assert r.returncode == 1, f"{name}: pins returned {r.returncode}\n{r.stdout[-3000:]}\n{r.stderr[-2000:]}"
