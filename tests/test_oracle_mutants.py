"""The oracle's pins catch the slips they are meant to catch.

Each case below plants one plausible mistake in a copy of the oracle's
source and runs the oracle's pins against the mutant: at least one must
fail.  The unmodified oracle passes the same pins, so a mutant that
survived would mean the pins leave that part of the oracle unchecked.

* C++ kernels of the oracle (a dropped key segment, a flipped sign, a wrong
  GQA index, a transposed operand, the scale applied twice, a wrong
  tie-break, an off-by-one in the refresh rule, ...): the mutated copy is
  built into a temporary library and run against every pin of
  tests/test_oracle_pins.py and the oracle fixtures of tests/test_golden.py.
* Python parts (the rollback decoder, the Algorithm 1 driver, the
  staleness bound): the mutated module source is executed into a fresh
  module, the one mutated function is patched into the oracle's module, and
  tests/test_decoder_oracle.py, tests/test_trajectory_oracle.py and
  tests/test_staleness_oracle.py run against it.

Every planted change keeps every memory access in bounds (the transposed
reads index an [D, N] view of the same N x D buffer), so a mutant can only
compute a wrong value, never crash the test process.  CPU only.
"""
import inspect
import os
import types

import pytest

from oracle import oracle as O
from oracle import staleness as OS
from oracle import trajectory as OT

import test_decoder_oracle
import test_golden
import test_oracle_pins
import test_staleness_oracle
import test_trajectory_oracle

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
    ("cur_prob_gating_inverted", "if (cur_tokens && !masked &&", "if (cur_tokens && masked &&"),
    ("margin_from_logits", "margin[r] = p[t1] - (t2 >= 0 ? p[t2] : 0.0);",
     "margin[r] = zr[t1] - (t2 >= 0 ? zr[t2] : 0.0);"),
    ("refresh_keeps_old_cache", "if (refresh && k_cache != k_new) {", "if (false) {"),
    ("cleared_flag_recomputes_prompt_rows", "const int32_t begin = refresh ? 0 : P;", "const int32_t begin = 0;"),
    ("lse_layout_transposed", "if (lse) lse[((size_t)b * Hq + h) * M + i] = l;",
     "if (lse) lse[((size_t)b * M + i) * Hq + h] = l;"),
    ("age_never_grows", "age[b] = (int32_t)age_t;", "age[b] = age[b];"),
    ("age_not_reset_on_refresh", "age[b] = 0;", "age[b] = (int32_t)age_t;"),
]


# (module, function, name, original text, planted text) for the Python parts.
PY_MUTANTS = [
    (O, "decoder_update", "accept_strict", "if mp[b, i] >= tau_accept:", "if mp[b, i] > tau_accept:"),
    (O, "decoder_update", "remask_wrong_direction", "elif cp[b, i] < tau_remask:", "elif cp[b, i] > tau_remask:"),
    (O, "decoder_update", "remask_inclusive", "elif cp[b, i] < tau_remask:", "elif cp[b, i] <= tau_remask:"),
    (O, "decoder_update", "progress_highest_index_on_ties", "if mp[b, i] > best:", "if mp[b, i] >= best:"),
    (O, "decoder_update", "progress_rule_dropped", "if not accepted and best_i >= 0:", "if False:"),
    (OT, "run", "cached_step_reads_fresh_prompt",
     'O.attn_step(x["q_all"][:, P:], x["k_cache"], x["v_cache"],',
     'O.attn_step(x["q_all"][:, P:], x["k_new"], x["v_new"],'),
    (OT, "run", "anchor_not_carried", "dist, flag, g_anchor, age = O.should_refresh(",
     "dist, flag, _anchor, age = O.should_refresh("),
    (OT, "run", "redrawn_query_rows_offset", 'x["q_all"][bidx, P + pos] = _f64(rows["q"])',
     'x["q_all"][bidx, pos] = _f64(rows["q"])'),
    (OT, "run", "response_k_not_redrawn", 'x["k_resp"][bidx, pos] = _f64(rows["k"])',
     'x["k_resp"][bidx, pos] = x["k_resp"][bidx, pos]'),
    (OT, "run", "refresh_ignores_flags", "scale, flags=flag,", "scale, flags=None,"),
    (OS, "gamma", "gamma_drops_value_term", "return b_e * alpha_row * (av + scale * qn * ak * vmax)",
     "return b_e * alpha_row * (scale * qn * ak * vmax)"),
    (OS, "gamma", "gamma_drops_key_term", "return b_e * alpha_row * (av + scale * qn * ak * vmax)",
     "return b_e * alpha_row * av"),
    (OS, "curve", "curve_compares_cached_with_itself", "o_fresh, _ = O.attn_step(q, kf, vf, kg, vg, scale)",
     "o_fresh, _ = O.attn_step(q, kc, vc, kg, vg, scale)"),
    (OS, "curve", "bound_linear_in_distance", "gam * math.sqrt(d)", "gam * d"),
]

PIN_MODULES = (test_oracle_pins, test_golden)
PY_PIN_MODULES = (test_decoder_oracle, test_trajectory_oracle, test_staleness_oracle)


def _pins(modules=PIN_MODULES):
    """Every oracle pin as (label, zero-argument callable), parametrized cases
    expanded; tests that need fixtures (the GPU ones) are left out."""
    out = []
    for mod in modules:
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


def _caught_by(pins, first=False):
    failed = []
    for label, call in pins:
        try:
            call()
        except AssertionError:
            failed.append(label)
            if first:
                break
    return failed


def test_pin_battery_is_complete():
    labels = [label for label, _ in _pins()]
    assert sum(label.startswith("test_oracle_pins.") for label in labels) >= 25
    assert sum(label.startswith("test_golden.") for label in labels) >= 3
    py = [label for label, _ in _pins(PY_PIN_MODULES)]
    assert len(py) >= 16


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
    caught = _caught_by(_pins(), first=True)
    assert caught, f"no oracle pin fails when the oracle has the slip '{name}'"


def _mutated_function(mod, fn_name, orig, planted):
    """fn_name from a fresh copy of mod whose source has orig replaced."""
    with open(mod.__file__) as f:
        src = f.read()
    fn_src = inspect.getsource(getattr(mod, fn_name))
    assert src.count(orig) == 1 and fn_src.count(orig) == 1, "mutation site is not unique in its function"
    fresh = types.ModuleType(mod.__name__ + "_mutant")
    fresh.__file__ = mod.__file__
    exec(compile(src.replace(orig, planted), mod.__file__, "exec"), fresh.__dict__)
    return getattr(fresh, fn_name)


@pytest.mark.parametrize("mod,fn_name,name,orig,planted", PY_MUTANTS, ids=[m[2] for m in PY_MUTANTS])
def test_planted_slip_in_python_oracle_fails_a_pin(mod, fn_name, name, orig, planted, monkeypatch):
    monkeypatch.setattr(mod, fn_name, _mutated_function(mod, fn_name, orig, planted))
    caught = _caught_by(_pins(PY_PIN_MODULES), first=True)
    assert caught, f"no oracle pin fails when {mod.__name__}.{fn_name} has the slip '{name}'"
