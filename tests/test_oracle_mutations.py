"""Mutation tests of the oracle's pins.

The pins in test_oracle_pins.py are only worth something if a plausible
mistake anywhere in the oracle fails at least one of them. Each case below
plants one such mistake (a dropped term, a wrong sign, index, divisor or
operand, a reversed ordering) in a copy of oracle/dc_oracle.c, compiles the
copy, and runs the pin file against it in a child process: the pins must fail.
The unmodified copy, compiled the same way, must pass them.

Only test_oracle_pins.py runs against the copies, and without the one pin that
checks a part of the oracle against another part (the global token mode with a
single row against the per-row oracle): a mistake must be caught by a library
routine, a closed form, an invariant or brute force. The stored tiny-workload
values in tests/golden/ come from the oracle itself, so they would catch any
change of its arithmetic and prove nothing about the pins.

Every planted mistake keeps memory accesses in bounds, so a copy fails on its
values, not on a crash.
"""

import os
import re
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
ORACLE = os.path.join(ROOT, "oracle")
PINS = os.path.join("tests", "test_oracle_pins.py")
# compares the global token mode with the per-row oracle: not independent of it
CROSS_CHECK = PINS + "::test_global_mode_with_one_row_is_the_row_oracle"

# (name, text in dc_oracle.c, replacement, occurrences to replace: 0 = all)
MUTANTS = [
    # attention and entropy (Sec. 3.1.1 entropy; Sec. 3.1 Reward, normalised weights)
    ("softmax scale 1/d instead of 1/sqrt(d)",
     "double scale = 1.0 / sqrt((double)d);", "double scale = 1.0 / (double)d;", 1),
    ("softmax denominator without the max shift",
     "l += exp(s[i] - m);", "l += exp(s[i]);", 1),
    ("entropy with the wrong sign",
     "if (ai > 0.0) H -= ai * log(ai);", "if (ai > 0.0) H += ai * log(ai);", 1),
    ("entropy in base 2",
     "if (ai > 0.0) H -= ai * log(ai);", "if (ai > 0.0) H -= ai * log2(ai);", 1),
    ("output weights the keys instead of the values",
     "+= ai * V[(size_t)i * d + c];", "+= ai * K[(size_t)i * d + c];", 1),
    ("the running max misses the last key",
     "if (s[i] > m) m = s[i];", "if (s[i] > m && i + 1 < n) m = s[i];", 1),
    # features (Sec. 3.1.1 State Space)
    ("alpha averaged over G + 1 heads",
     "    mean /= G;\n", "    mean /= G + 1;\n", 1),
    ("alpha is the first head's mass only",
     "for (int h = 0; h < G; ++h) mean += a[(size_t)i * G + h];",
     "for (int h = 0; h < 1; ++h) mean += a[(size_t)i * G + h];", 1),
    ("sigma as the sample variance",
     "    var /= G;\n", "    var /= (G > 1 ? G - 1 : 1);\n", 1),
    ("sigma as the standard deviation",
     "    var /= G;\n", "    var = sqrt(var / G);\n", 1),
    ("|v_i| squared (no square root)",
     "    vn = sqrt(vn);\n", "", 1),
    ("|v_i| of the key instead of the value",
     "vn += r->v[(size_t)i * d + c] * r->v[(size_t)i * d + c];",
     "vn += r->k[(size_t)i * d + c] * r->k[(size_t)i * d + c];", 1),
    ("H_i unnormalised (S_i instead of S_i / Z_i)",
     "double Hi = Z > 0.0 ? S / Z : 0.0;", "double Hi = S;", 1),
    ("H_i weights every head by head 0's entropy",
     "S += we->a[(size_t)j * G + h] * we->H[h];", "S += we->a[(size_t)j * G + h] * we->H[0];", 1),
    ("H_i window leaves out the current query",
     "      if (j < 0) continue; /* not yet in the cache at that step */",
     "      if (j < 0 || qi == newest_entry) continue;", 1),
    ("H_i window holds one query fewer",
     "if (r->win_count < r->w) r->win_count += 1;",
     "if (r->win_count < r->w - 1) r->win_count += 1;", 1),
    ("H_i keyed by slot instead of position",
     "int j = find_pos(we->pos, we->n, r->pos[i]);", "int j = i < we->n ? i : -1;", 1),
    ("prior window sums keep only the current query",
     "        if (qi != newest_entry) {\n          Zp", "        if (qi == newest_entry) {\n          Zp", 1),
    ("pos_i by slot rank instead of position",
     "double posn = (double)r->pos[i] / pos_den;", "double posn = (double)i / pos_den;", 1),
    ("pos_i normalised by the row length",
     "int64_t newest = r->pos[n - 1];\n  double pos_den = (double)(newest > 1 ? newest : 1);",
     "int64_t newest = r->pos[n - 1];\n  double pos_den = (double)(n > 1 ? n : 1);", 1),
    ("cumulative alpha not accumulated",
     "r->acc[i] += mean;", "r->acc[i] = mean;", 1),
    ("cumulative alpha of a new token not reset (a reused slot keeps the old mass)",
     "  r->acc[i] = 0.0;\n  r->n += 1;\n", "  r->n += 1;\n", 1),
    ("sigma around the cumulative alpha instead of this step's mean",
     "double dv = a[(size_t)i * G + h] - mean;", "double dv = a[(size_t)i * G + h] - alpha;", 1),
    ("entropy term 0 * ln 0 not taken as 0",
     "if (ai > 0.0) H -= ai * log(ai);", "H -= ai * log(ai);", 1),
    ("features in the wrong order (sigma and |v| swapped)",
     "x[(size_t)i * 5 + 1] = vn;\n    x[(size_t)i * 5 + 2] = var;\n    x[(size_t)i * 5 + 3] = Hi;",
     "x[(size_t)i * 5 + 1] = var;\n    x[(size_t)i * 5 + 2] = vn;\n    x[(size_t)i * 5 + 3] = Hi;", 1),
    # policy MLP (Sec. 3.1.2; App. D)
    ("first layer weights transposed",
     "acc += (double)W1[j * 5 + c] * xt[c];", "acc += (double)W1[c * hidden + j] * xt[c];", 1),
    ("LayerNorm mean not divided by the width",
     "      mu /= hidden;\n", "", 1),
    ("first layer bias dropped",
     "double acc = (double)b1[j];", "double acc = 0.0;", 1),
    ("LayerNorm with the unbiased variance",
     "      var /= hidden;\n", "      var /= hidden - 1;\n", 1),
    ("LayerNorm eps 1e-3",
     "1.0 / sqrt(var + 1e-5)", "1.0 / sqrt(var + 1e-3)", 1),
    ("LayerNorm gain and shift swapped",
     "* inv * (double)gamma[j] + (double)beta[j];", "* inv * (double)beta[j] + (double)gamma[j];", 1),
    ("ReLU dropped",
     "out += (double)w2[j] * (h[j] > 0.0 ? h[j] : 0.0);", "out += (double)w2[j] * h[j];", 1),
    ("output bias dropped",
     "double out = b2;", "double out = 0.0;", 1),
    # argtop_B and prune (Algorithm 1)
    ("keeps the lowest scores",
     "if (!nx && x->s != y->s) return x->s > y->s ? -1 : 1;",
     "if (!nx && x->s != y->s) return x->s < y->s ? -1 : 1;", 1),
    ("ties go to the higher position",
     "return (x->p > y->p) - (x->p < y->p);", "return (x->p < y->p) - (x->p > y->p);", 1),
    ("NaN ranks above every number",
     "if (nx != ny) return nx ? 1 : -1;", "if (nx != ny) return nx ? -1 : 1;", 1),
    ("one survivor too few",
     "int keep_n = budget < n ? budget : n;\n  if (keep_n < 0) keep_n = 0;\n  rank_item* it = (rank_item*)malloc(sizeof(rank_item) * (size_t)(n > 0 ? n : 1));\n  for (int i = 0; i < n; ++i) {\n    it[i].s = scores_f32 ? (double)scores_f32[i] : r->score[i];",
     "int keep_n = budget < n ? budget : n - 1;\n  if (keep_n < 0) keep_n = 0;\n  rank_item* it = (rank_item*)malloc(sizeof(rank_item) * (size_t)(n > 0 ? n : 1));\n  for (int i = 0; i < n; ++i) {\n    it[i].s = scores_f32 ? (double)scores_f32[i] : r->score[i];", 1),
    ("prune drops the cumulative mass of moved tokens",
     "      r->acc[w] = r->acc[i];\n", "", 1),
    ("prune moves the keys but not the values",
     "      memmove(r->vb + (size_t)w * d, r->vb + (size_t)i * d, sizeof(uint16_t) * d);\n", "", 1),
    ("positions restart at the slot index",
     "  r->pos[i] = r->seen;\n", "  r->pos[i] = i;\n", 1),
    # heuristic scorers (Sec. 2, Sec. 4)
    ("StreamingLLM keeps one sink too many",
     "score[i] = r->pos[i] < (int64_t)n_sinks ?", "score[i] = r->pos[i] <= (int64_t)n_sinks ?", 1),
    ("H2O scores the latest step's mass only",
     "for (int i = 0; i < r->n; ++i) score[i] = r->acc[i];",
     "for (int i = 0; i < r->n; ++i) score[i] = r->acc[i] / (double)(r->seen - r->pos[i]);", 1),
    # training side (App. C)
    ("log Z items added lowest k first (an item counted twice)",
     "for (int k = B; k >= 1; --k) e[k] = log_add(e[k], y + e[k - 1]);",
     "for (int k = 1; k <= B; ++k) e[k] = log_add(e[k], y + e[k - 1]);", 1),
    ("log Z without the temperature",
     "const double y = s[i] / tau;", "const double y = s[i];", 1),
    ("log-add without the 1 +",
     "return m + log1p(exp(-fabs(a - b)));", "return m + log(exp(-fabs(a - b)) + 1e-300);", 1),
    ("Gumbel noise subtracted",
     "volatile float v = y + g[i];", "volatile float v = y - g[i];", 1),
    ("Gumbel ties go to the higher index",
     "return (a->i > b->i) - (a->i < b->i);", "return (a->i < b->i) - (a->i > b->i);", 1),
    # global token mode (Sec. 3.1.1: features pooled over heads and layers)
    ("global alpha averaged over rows only",
     "    mean /= N;\n", "    mean /= R;\n", 1),
    ("global |v| summed over rows",
     "    vn /= R;\n", "", 1),
    ("global entropy weight from row 0",
     "e->sa[i] += ah * Hh[(size_t)r * G + h];", "e->sa[i] += ah * Hh[h];", 1),
    ("global sigma as the sample variance",
     "    var /= N;\n", "    var /= (N > 1 ? N - 1 : 1);\n", 1),
    ("global window leaves out the current step",
     "      if (j < 0) continue;\n      Z += we->za[j];", "      if (j < 0 || qi == newest_entry) continue;\n      Z += we->za[j];", 1),
    ("global window keyed by slot instead of position",
     "const int j = find_pos(we->pos, we->n, s->pos[i]);", "const int j = i < we->n ? i : -1;", 1),
    ("global prior window sums keep only the current step",
     "      if (qi != newest_entry) {\n        Zp += we->za[j];", "      if (qi == newest_entry) {\n        Zp += we->za[j];", 1),
    ("global pos_i by slot rank instead of position",
     "x[(size_t)i * 5 + 4] = (double)s->pos[i] / pos_den;", "x[(size_t)i * 5 + 4] = (double)i / pos_den;", 1),
    ("global cumulative alpha not accumulated",
     "s->acc[i] += mean;", "s->acc[i] = mean;", 1),
    ("global append reads the tokens as [T][R] instead of [R][T]",
     "seq_put(s, r, s->n, k + ((size_t)r * T + t) * s->d, v + ((size_t)r * T + t) * s->d);",
     "seq_put(s, r, s->n, k + ((size_t)t * s->R + r) * s->d, v + ((size_t)t * s->R + r) * s->d);", 1),
    ("global step gives every row the first row's query",
     "qd[i] = bf16_to_double(q[(size_t)r * G * d + i]);", "qd[i] = bf16_to_double(q[i]);", 1),
    ("global step gives every row the first row's new key",
     "seq_put(s, r, s->n, k_new + (size_t)r * d, v_new + (size_t)r * d);",
     "seq_put(s, r, s->n, k_new, v_new + (size_t)r * d);", 1),
    ("global prune moves row 0 only",
     "      for (int r = 0; r < s->R; ++r) {\n        const size_t src",
     "      for (int r = 0; r < 1; ++r) {\n        const size_t src", 1),
]


def _mutate(text: str, old: str, new: str, count: int) -> str:
    found = text.count(old)
    assert found >= 1, f"snippet not found in dc_oracle.c: {old!r}"
    if count:
        assert found == count, f"snippet found {found} times, expected {count}: {old!r}"
    return text.replace(old, new)


def _run_pins(workdir: str, name: str, source: str) -> tuple[int, str]:
    """Compiles `source` as the oracle and runs the pin file against it.
    Returns (pytest exit code, the first failing test or the output tail)."""
    d = os.path.join(workdir, name)
    os.makedirs(d)
    shutil.copy(os.path.join(ORACLE, "dc_oracle.h"), d)
    src = os.path.join(d, "dc_oracle.c")
    with open(src, "w") as f:
        f.write(source)
    so = os.path.join(d, "libdc_oracle.so")
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fno-fast-math", "-o", so, src,
                           "-lm"])
    env = dict(os.environ, DC_ORACLE_LIB=so)
    p = subprocess.run([sys.executable, "-m", "pytest", PINS, "--deselect", CROSS_CHECK, "-x", "-q", "-p",
                        "no:cacheprovider", "-m", "not gpu"],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    m = re.search(r"FAILED (\S+)", p.stdout)
    return p.returncode, m.group(1) if m else p.stdout[-400:]


@pytest.fixture(scope="module")
def results(tmp_path_factory):
    with open(os.path.join(ORACLE, "dc_oracle.c")) as f:
        text = f.read()
    jobs = {"unmodified": text}
    for i, (name, old, new, count) in enumerate(MUTANTS):
        jobs[f"m{i:02d}"] = _mutate(text, old, new, count)
    work = str(tmp_path_factory.mktemp("oracle_mutants"))
    with ThreadPoolExecutor(max_workers=max(2, min(8, os.cpu_count() or 2))) as ex:
        futs = {k: ex.submit(_run_pins, work, k, src) for k, src in jobs.items()}
        return {k: f.result() for k, f in futs.items()}


def test_unmodified_copy_passes_the_pins(results):
    code, detail = results["unmodified"]
    assert code == 0, detail


@pytest.mark.parametrize("i", range(len(MUTANTS)), ids=[m[0] for m in MUTANTS])
def test_planted_mistake_fails_a_pin(results, i):
    code, detail = results[f"m{i:02d}"]
    # exit code 1: tests ran and at least one failed (not a collection or usage error)
    assert code == 1, f"the pins did not catch: {MUTANTS[i][0]} (exit {code}; {detail})"
