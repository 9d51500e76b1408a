"""Pin strength: each plausible mistake planted in a copy of the oracle (on the
CPU, compiled to a temporary library) must make at least one pin fail.

The mutations are the slips a reader of Eq. 1-3, Sec. 4.3 and Sec. 4.4 could
make: an off-by-one query or candidate row, a dropped norm, a flipped tie-break,
a non-strict comparison, the wrong attention key, the wrong bonus row.  Every
mutation keeps all memory accesses inside the inputs.
"""
import inspect
import os
import subprocess

import pytest

import oracle
from tests import test_oracle_golden as golden
from tests import test_oracle_pins as pins

SRC = os.path.join(os.path.dirname(oracle.__file__), "pldp_oracle.c")

MUTANTS = [
    ("query row H_t instead of H_{t-1}",
     "(t - 1) * d;   /* H_{t-1} */", "t * d;   /* H_{t-1} */"),
    ("candidate row H_j instead of H_{j-1}",
     "(j - 1) * d;   /* H_{j-1} */", "j * d;   /* H_{j-1} */"),
    ("cosine without the candidate norm",
     "return dot / sqrt(na * nb);", "return dot / sqrt(nb * nb);"),
    ("cosine zero-norm guard dropped",
     "if (na == 0.0 || nb == 0.0) return 0.0;", ""),
    ("hidden tie goes to the larger position",
     "if (j >= 1 && j < t && s > threshold) {\n                if (bj < 0 || s > bs || (s == bs && j < bj))",
     "if (j >= 1 && j < t && s > threshold) {\n                if (bj < 0 || s > bs || (s == bs && j > bj))"),
    ("attention tie goes to the larger position",
     "if (j >= 0 && j < t) {\n                if (bj < 0 || s > bs || (s == bs && j < bj))",
     "if (j >= 0 && j < t) {\n                if (bj < 0 || s > bs || (s == bs && j > bj))"),
    ("threshold not strict",
     "s > threshold", "s >= threshold"),
    ("j = 0 scored against H_0 and eligible",
     "if (j >= 1 && j < t) {\n                int64_t row_cand  = (int64_t)b * seq_stride + (j - 1) * d;",
     "if (j >= 0 && j < t) {\n                int64_t row_cand  = (int64_t)b * seq_stride + (j > 0 ? j - 1 : 0) * d;"),
    ("candidate search allows j = t",
     "for (int64_t j = 0; j < t; ++j) {", "for (int64_t j = 0; j <= t; ++j) {"),
    ("shortest n-gram first",
     "for (int n = ngram_max; n >= ngram_min; --n) {", "for (int n = ngram_min; n <= ngram_max; ++n) {"),
    ("n-gram compares one token too few",
     "for (int k = 0; k < n; ++k)\n        if (x[j - k] != x[t - k]) return 0;",
     "for (int k = 1; k < n; ++k)\n        if (x[j - k] != x[t - k]) return 0;"),
    ("overflow flag off by one",
     "if (count > C_cap && status)", "if (count > C_cap + 1 && status)"),
    ("attention key j+1 instead of j",
     "(int64_t)r * row_stride + j);", "(int64_t)r * row_stride + j + 1);"),
    ("attention max replaced by sum",
     "if (agg == ORC_AGG_MAX) { if (a > s) s = a; }", "if (agg == ORC_AGG_MAX) { s += a; }"),
    ("draft starts at x_{j*} instead of x_{j*+1}",
     "ids[(int64_t)b * ids_stride + js + 1 + i]", "ids[(int64_t)b * ids_stride + js + i]"),
    ("argmax keeps the last of equal maxima",
     "if (x > best) { best = x; bi = (int32_t)v; }", "if (x >= best) { best = x; bi = (int32_t)v; }"),
    ("bonus token from the row after the whole draft",
     "int32_t bonus = tok[n];", "int32_t bonus = tok[d];"),
    ("kv_keep counts the bonus token",
     "kv_keep_len[b] = (int32_t)(L + n);", "kv_keep_len[b] = (int32_t)(L + n + 1);"),
    ("accept ignores the first draft token",
     "for (int64_t i = 0; i < d; ++i) {\n        if (draft[(int64_t)b * K + i] != tok[i]) { n = i; break; }",
     "for (int64_t i = 1; i < d; ++i) {\n        if (draft[(int64_t)b * K + i] != tok[i]) { n = i; break; }"),
    ("averaged-ranking tie goes to the larger position",
     "/* eligible: the smallest j wins a tie */\n                if (bj < 0 || s > bs || (s == bs && j < bj))",
     "/* eligible: the smallest j wins a tie */\n                if (bj < 0 || s > bs || (s == bs && j > bj))"),
    ("averaging window one row too long",
     "int64_t lo = p - m + 1;\n    if (lo < 0) lo = 0;", "int64_t lo = p - m;\n    if (lo < 0) lo = 0;"),
    ("averaging window misses the row averaged",
     "for (int64_t r = lo; r <= p; ++r)", "for (int64_t r = lo; r < p; ++r)"),
    ("identification overlap ignores the copied token itself",
     "while (k < max_suffix && j - k >= 0 && x[j - k] == x[p - k]) ++k;",
     "while (k < max_suffix && j - k - 1 >= 0 && x[j - k - 1] == x[p - k - 1]) ++k;"),
    ("identification tie goes to the larger position",
     "if (k > best_ov) { best_ov = k; rs = j; }", "if (k >= best_ov) { best_ov = k; rs = j; }"),
    ("identification row argmax keeps the last maximum",
     "if (v > mx) { mx = v; arg = key; }", "if (v >= mx) { mx = v; arg = key; }"),
    ("identification looks at the generated position's own key",
     "for (int64_t key = 1; key < p; ++key) {", "for (int64_t key = 1; key <= p; ++key) {"),
    ("sampling draws where the cumulative sum only reaches u",
     "if (c > target) { y = (int32_t)v; break; }", "if (c >= target) { y = (int32_t)v; break; }"),
    ("sampling multiplies by the temperature",
     "double w = exp((orc_load(logits, dtype, row + v) - m) / temperature);",
     "double w = exp((orc_load(logits, dtype, row + v) - m) * temperature);"),
    ("sampling takes the next position's uniform",
     "double u = (double)uniforms[(int64_t)b * (K + 1) + i];",
     "double u = (double)uniforms[(int64_t)b * (K + 1) + (i + 1) % (K + 1)];"),
    ("sampling bonus from the argmax instead of the draw",
     "yv[i] = y;", "yv[i] = (i == K) ? 0 : y;"),
]


def _pin_calls(orc):
    """Every pin test, as a zero-argument callable."""
    calls = []
    for mod in (golden, pins):
        for name, fn in inspect.getmembers(mod, inspect.isfunction):
            if not name.startswith("test_"):
                continue
            params = list(inspect.signature(fn).parameters)
            marks = getattr(fn, "pytestmark", [])
            grids = [dict()]
            for m in marks:
                if m.name != "parametrize":
                    continue
                names = [s.strip() for s in m.args[0].split(",")]
                vals = m.args[1]
                grids = [dict(g, **dict(zip(names, v if len(names) > 1 else (v,))))
                         for g in grids for v in vals]
            for g in grids:
                kw = {k: v for k, v in g.items()}
                if "orc" in params:
                    kw["orc"] = orc
                calls.append((name, lambda fn=fn, kw=kw: fn(**kw)))
    return calls


@pytest.mark.parametrize("desc,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_mutant_is_caught(tmp_path, desc, old, new):
    src = open(SRC).read()
    assert src.count(old) == 1, f"mutation anchor not unique/present: {desc}"
    mpath = tmp_path / "mutant.c"
    mpath.write_text(src.replace(old, new))
    so = tmp_path / "libmutant.so"
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", str(mpath), "-o", str(so), "-lm"])
    prev = oracle.use_library(str(so))
    try:
        failed = []
        for name, call in _pin_calls(oracle):
            try:
                call()
            except AssertionError:
                failed.append(name)
                break
        assert failed, f"no pin catches the mutation: {desc}"
    finally:
        oracle.restore_library(prev)
