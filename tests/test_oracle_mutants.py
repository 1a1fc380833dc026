"""The oracle's pins catch the slips they are meant to catch.

Each case below plants one plausible mistake in a copy of the oracle's C++
source (a dropped key segment, a flipped sign, a wrong GQA index, a
transposed operand, the scale applied twice, a wrong tie-break, an
off-by-one in the refresh rule, ...), builds that copy into a temporary
library, and runs every pin of tests/test_oracle_pins.py and the oracle
fixtures of tests/test_golden.py against it: at least one must fail.  The
unmodified oracle passes the same pins in those files, so a mutant that
survived would mean the pins leave that part of the oracle unchecked.

Every planted change keeps every memory access in bounds (the transposed
reads index an [D, N] view of the same N x D buffer), so a mutant can only
compute a wrong value, never crash the test process.  CPU only.
"""
import inspect
import os

import pytest

from oracle import oracle as O

import test_golden
import test_oracle_pins

# (name, original text, planted text): the original must occur exactly once.
MUTANTS = [
    ("drop_prompt_segment",
     "for (int j = 0; j < P; ++j) {\n    const size_t src = (((size_t)b * P + j)",
     "for (int j = 0; j < 0; ++j) {\n    const size_t src = (((size_t)b * P + j)"),
    ("drop_response_segment",
     "for (int j = 0; j < G; ++j) {\n    const size_t src = (((size_t)b * G + j)",
     "for (int j = 0; j < 0; ++j) {\n    const size_t src = (((size_t)b * G + j)"),
    ("exp_sign_flipped", "e[j] = std::exp(s[j] - m);", "e[j] = std::exp(m - s[j]);"),
    ("gqa_modulo_index", "const int kvh = h / group;", "const int kvh = h % Hkv;"),
    ("k_transposed", "dot += q[c] * kcat[(size_t)j * d + c];", "dot += q[c] * kcat[(size_t)c * n_keys + j];"),
    ("v_transposed", "out[c] += p[j] * vcat[(size_t)j * d + c];",
     "out[c] += p[j] * vcat[(size_t)c * n_keys + j];"),
    ("scale_applied_twice", "s[j] = scale * dot;", "s[j] = scale * scale * dot;"),
    ("softmax_not_normalised", "p[j] = e[j] / sum;", "p[j] = e[j];"),
    ("lse_missing_log", "*lse = m + std::log(sum);", "*lse = m + sum;"),
    ("top1_highest_index_on_ties", "if (t1 < 0 || zr[j] > zr[t1]) t1 = j;",
     "if (t1 < 0 || zr[j] >= zr[t1]) t1 = j;"),
    ("top2_skips_ties", "if (j == t1) continue;", "if (zr[j] == zr[t1]) continue;"),
    ("distance_strict", "const bool f = (d >= K) ||", "const bool f = (d > K) ||"),
    ("age_off_by_one", "(max_age > 0 && age_t >= max_age)", "(max_age > 0 && age_t > max_age)"),
    ("cached_step_reads_fresh_prompt",
     "const double* kp = refresh ? k_new + b * per_seq : k_cache + b * per_seq;\n"
     "    const double* vp = refresh ? v_new + b * per_seq : v_cache + b * per_seq;",
     "const double* kp = k_new + b * per_seq;\n"
     "    const double* vp = v_new + b * per_seq;"),
    ("anchor_not_updated", "g_anchor[(size_t)b * G + i] = g_cur[(size_t)b * G + i];", "(void)0;"),
]


def _pins():
    """Every oracle pin as (label, zero-argument callable), parametrized cases
    expanded; tests that need fixtures (the GPU ones) are left out."""
    out = []
    for mod in (test_oracle_pins, test_golden):
        for name, fn in sorted(vars(mod).items()):
            if not name.startswith("test_") or not callable(fn):
                continue
            params = list(inspect.signature(fn).parameters)
            marks = [m for m in getattr(fn, "pytestmark", []) if m.name == "parametrize"]
            if not params:
                out.append((f"{mod.__name__}.{name}", fn))
                continue
            if len(marks) != 1 or any(m.name == "gpu" for m in getattr(fn, "pytestmark", [])):
                continue
            argnames = [a.strip() for a in marks[0].args[0].split(",")]
            if sorted(argnames) != sorted(params):
                continue
            for k, vals in enumerate(marks[0].args[1]):
                vals = vals if len(argnames) > 1 else (vals,)
                kw = dict(zip(argnames, vals))
                out.append((f"{mod.__name__}.{name}[{k}]", lambda fn=fn, kw=kw: fn(**kw)))
    return out


def _caught_by(pins):
    failed = []
    for label, call in pins:
        try:
            call()
        except AssertionError:
            failed.append(label)
    return failed


def test_pin_battery_is_complete():
    labels = [label for label, _ in _pins()]
    assert sum(label.startswith("test_oracle_pins.") for label in labels) >= 25
    assert sum(label.startswith("test_golden.") for label in labels) >= 3


@pytest.mark.parametrize("name,orig,planted", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_planted_slip_fails_a_pin(name, orig, planted, tmp_path, monkeypatch):
    with open(O._SRC) as f:
        src = f.read()
    assert src.count(orig) == 1, f"mutation site for {name} is not unique in the oracle source"
    path = os.path.join(tmp_path, "archer_oracle.cpp")
    with open(path, "w") as f:
        f.write(src.replace(orig, planted))
    monkeypatch.setattr(O, "_SRC", path)
    monkeypatch.setattr(O, "_BUILD", os.path.join(tmp_path, "_build"))
    monkeypatch.setattr(O, "_lib", None)
    caught = _caught_by(_pins())
    assert caught, f"no oracle pin fails when the oracle has the slip '{name}'"
