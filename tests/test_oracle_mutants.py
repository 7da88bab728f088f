"""The oracle's pins catch plausible mistakes.

Each case plants one mistake in a scratch copy of the oracle's C source (the
committed file is never touched), builds it into the test's temporary folder and
runs tests/test_oracle_pins.py against that build in a subprocess: at least one
pin must fail. The mistakes are those a restatement of Sec. 4.2-4.4 could
plausibly make: a softmax axis or scale, a dropped normalisation, a de-meaning
left out, a tie rule reversed, an off-by-one causal range, the wrong key/value
head, a sample instead of a population variance, a compaction range cut short.

Not listed: replacing the strict r_j > Mean(r) of Sec. 4.2 by >=. The two differ
only when some r_j equals the mean exactly while the others do not; when every
r_j is equal, the empty-T fallback (all rows) gives the same set as >=. Such an
exact tie is not reachable from continuous inputs in double precision, so no
pin can tell the two apart.
"""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
ORACLE_SRC = os.path.join(ROOT, "oracle", "provip_oracle.c")
PINS = os.path.join(ROOT, "tests", "test_oracle_pins.py")

# (what the mistake is, text in the oracle source, replacement)
MUTANTS = [
    ("crit text: column sums into the row index (softmax over the other axis)",
     "for (int j = 0; j < n; ++j) r[j] += exp(row[j] - mx) / z;",
     "for (int j = 0; j < n; ++j) r[i] += exp(row[j] - mx) / z;"),
    ("crit text: a 1/sqrt(d) scale the paper does not write",
     "row[j] = dot_d(E + (size_t)i * d, E + (size_t)j * d, d);",
     "row[j] = dot_d(E + (size_t)i * d, E + (size_t)j * d, d) / sqrt((double)d);"),
    ("crit text: r not divided by N_t",
     "for (int j = 0; j < n; ++j) r[j] /= (double)n;", ""),
    ("crit text: no fallback for an empty T",
     "    for (int j = 0; j < n; ++j) mask[j] = 1;\n    free(row);", "    ;\n    free(row);"),
    ("relevance: no de-meaning",
     "double mh = M[(size_t)a * nv + j] - mu;", "double mh = M[(size_t)a * nv + j];"),
    ("relevance: row mean divided by |T| instead of N_v",
     "mu /= (double)nv;", "mu /= (double)nT;"),
    ("relevance: last critical row instead of the max",
     "if (mh > p[j]) p[j] = mh;", "p[j] = mh;"),
    ("relevance: visual norm left out of the cosine",
     "return dot_d(a, b, d) / (na * nb);", "return dot_d(a, b, d) / na;"),
    ("relevance: min over rows instead of max",
     "for (int j = 0; j < nv; ++j) p[j] = -INFINITY;", "for (int j = 0; j < nv; ++j) p[j] = INFINITY;"),
    ("top-k: ties to the higher index",
     "return (a->i > b->i) - (a->i < b->i);", "return (a->i < b->i) - (a->i > b->i);"),
    ("top-k: indices not returned ascending",
     "qsort(idx, (size_t)k, sizeof(int), po_int_cmp);", ""),
    ("top-k: the k smallest",
     "if (a->s > b->s) return -1;\n    if (a->s < b->s) return 1;",
     "if (a->s > b->s) return 1;\n    if (a->s < b->s) return -1;"),
    ("merge: ties to the higher kept position",
     "if (c > bc) { bc = c; best = a; }", "if (c >= bc) { bc = c; best = a; }"),
    ("merge: dot product instead of cosine",
     "double c = cos_d(Ev + (size_t)j * d, Ev + (size_t)keep[a] * d, d);",
     "double c = dot_d(Ev + (size_t)j * d, Ev + (size_t)keep[a] * d, d);"),
    ("merge: mean divided by one too many",
     "merged[(size_t)a * d + e] /= (double)cnt[a];", "merged[(size_t)a * d + e] /= (double)(cnt[a] + 1);"),
    ("merge: second kept row never a candidate",
     "for (int a = 1; a < n1; ++a) {\n            double c", "for (int a = 2; a < n1; ++a) {\n            double c"),
    ("attention: no 1/sqrt(d_h)",
     "prob[k] = dot_d(q, K + ((size_t)k * Hkv + g) * dh, dh) * scale;",
     "prob[k] = dot_d(q, K + ((size_t)k * Hkv + g) * dh, dh);"),
    ("attention: key/value head h % H_kv instead of h / (H_q / H_kv)",
     "int g = h / (Hq / Hkv);", "int g = h % Hkv;"),
    ("head scores: a visual column at the row's own position left out",
     "S[i] += (col <= rows[j]) ? prob[col] : 0.0;", "S[i] += (col < rows[j]) ? prob[col] : 0.0;"),
    ("head scores: no mean over heads",
     "for (int i = 0; i < nv; ++i) v[i] += S[i] / (double)nh;", "for (int i = 0; i < nv; ++i) v[i] += S[i];"),
    ("head scores: no mean over text rows",
     "for (int i = 0; i < nv; ++i) v[i] /= (double)nr;", ""),
    ("confidence: sample variance instead of population",
     "C[h] += var / (double)nv;", "C[h] += var / (double)(nv - 1);"),
    ("confidence: max over rows instead of the sum",
     "C[h] += var / (double)nv;", "C[h] = fmax(C[h], var / (double)nv);"),
    ("confidence: mean over every causal key instead of the visual columns",
     "mean /= (double)nv;\n            double var", "mean /= (double)(rows[j] + 1);\n            double var"),
    ("compaction: first prefix row dropped",
     "for (int r = 0; r < vis_start; ++r) src[o++] = r;", "for (int r = 1; r < vis_start; ++r) src[o++] = r;"),
    ("compaction: last row dropped",
     "for (int r = vis_start + nv; r < seq_len; ++r) src[o++] = r;",
     "for (int r = vis_start + nv; r < seq_len - 1; ++r) src[o++] = r;"),
    ("batch: text rows shifted by one",
     "rows[j] = text_start[b] + j;", "rows[j] = text_start[b] + j + 1;"),
]

# run the pins in a fresh interpreter whose oracle module builds the scratch source
_RUNNER = ("import sys, oracle, pytest; oracle._SRC = sys.argv[1]; oracle._LIB_PATH = sys.argv[2]; "
           "sys.exit(pytest.main(['-q', '-x', '-m', 'not gpu', '-p', 'no:cacheprovider', sys.argv[3]]))")


@pytest.mark.parametrize("what,old,new", MUTANTS, ids=[m[0].split(":")[0] + f"-{i}" for i, m in enumerate(MUTANTS)])
def test_pins_catch_a_planted_mistake(tmp_path, what, old, new):
    src = open(ORACLE_SRC).read()
    assert src.count(old) == 1, f"mutation site not unique or missing: {what}"
    mutant = tmp_path / "provip_oracle_mutant.c"
    mutant.write_text(src.replace(old, new))
    r = subprocess.run([sys.executable, "-c", _RUNNER, str(mutant), str(tmp_path / "libmutant.so"), PINS],
                       cwd=ROOT, capture_output=True, text=True, timeout=600)
    # exit code 1: some pin failed (2 and up would be a build or collection error)
    assert r.returncode == 1, f"the pins did not catch: {what} (exit {r.returncode})\n{r.stdout[-3000:]}"
