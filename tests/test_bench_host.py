"""bench.py's host logic, on the CPU: the refresh fraction its CPU baseline
extrapolates with, the gate that drops a traffic figure once the kernel's
sources change, the peak table's fallback, and the whole-job rate."""
import importlib.util
import json
import os

import pytest

from paper_2608_08086_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bench():
    spec = importlib.util.spec_from_file_location("bench_host", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_refresh_fraction_follows_each_workloads_schedule(bench):
    # tiny: age cap 4 over 8 steps -> t = 4, 8; the long-prompt GQA workload:
    # age cap 16 over 32 steps -> t = 16, 32; the 32-layer trajectory: the
    # distance rule fires every third step (t = 3, 6, ..., 63: 21 of 64)
    assert bench.refresh_fraction(synth.WORKLOADS["tiny"]) == 2 / 8
    assert bench.refresh_fraction(synth.WORKLOADS["gqa_long"]) == 2 / 32
    assert bench.refresh_fraction(synth.WORKLOADS["traj32"]) == 21 / 64
    # no steps: nothing to refresh
    assert bench.refresh_fraction(synth.WORKLOADS["llada_layer"]) == 0.0


def test_traffic_figure_is_dropped_when_the_sources_change(bench, monkeypatch):
    key = ("attn_step", "gqa_long")
    ent = dict(bench.MEASURED_TRAFFIC[key])
    # a figure recorded for the sources as they are is reported
    monkeypatch.setitem(bench.MEASURED_TRAFFIC, key, dict(ent, sha16=bench._source_sha(ent["sources"])))
    assert bench.measured_traffic(*key) == ent["bytes"]
    monkeypatch.setitem(bench.MEASURED_TRAFFIC, key, dict(ent, sha16="0" * 16))
    assert bench.measured_traffic(*key) is None
    monkeypatch.setitem(bench.MEASURED_TRAFFIC, key, dict(ent, sources=["no_such_file.cu"]))
    assert bench.measured_traffic(*key) is None
    assert bench.measured_traffic("attn_step", "no_such_workload") is None


def test_traffic_entries_cover_the_compulsory_bytes(bench):
    # each recorded DRAM figure is at least what the launch must read:
    # cached step Q + prompt K/V + response K/V = 209.7 MB (the output write
    # partly stays in L2); scoring 16 x 512 x 152064 bf16 logits
    sh = synth.WORKLOADS["gqa_long"].shape
    reads = 2 * (sh.batch * sh.resp_len * sh.n_heads * sh.head_dim
                 + 2 * sh.batch * (sh.prompt_len + sh.resp_len) * sh.n_kv_heads * sh.head_dim)
    assert reads <= bench.MEASURED_TRAFFIC[("attn_step", "gqa_long")]["bytes"] <= reads + 2 * reads // 7
    # refresh: all N query rows and the fresh prompt K/V read, the output and
    # the cache (the fused rewrite) written; the copy reads the prompt again
    N = sh.prompt_len + sh.resp_len
    q_out = 2 * sh.batch * N * sh.n_heads * sh.head_dim
    kv_p = 2 * 2 * sh.batch * sh.prompt_len * sh.n_kv_heads * sh.head_dim
    kv_g = 2 * 2 * sh.batch * sh.resp_len * sh.n_kv_heads * sh.head_dim
    least = q_out + kv_p + kv_g + q_out // 2 + kv_p      # reads, and writes partly still in L2
    assert least <= bench.MEASURED_TRAFFIC[("attn_refresh", "gqa_long")]["bytes"] <= 2 * q_out + 3 * kv_p + kv_g
    logits = 2 * 16 * 512 * 152064
    assert logits <= bench.MEASURED_TRAFFIC[("scores", "gqa_long")]["bytes"] <= logits * 1.01


def test_peaks_fall_back_without_the_measured_table(bench, monkeypatch, tmp_path):
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    p, kind = bench.peaks()
    assert kind == "fallback" and p == bench.PEAKS_FALLBACK
    with open(os.path.join(tmp_path, "MEASURED_PEAKS.json"), "w") as f:
        json.dump({"hbm_gbs": 1.0, "bf16_tflops": 2.0, "bf16_tflops_sustained": 3.0}, f)
    p, kind = bench.peaks()
    assert kind == "measured" and p["hbm_gbs"] == 1.0


def test_whole_job_rate(bench):
    # 4 replicas x 20 steps in 500 ms -> 160 steps/s
    assert bench.whole_job_rate(4, 20, 500.0) == pytest.approx(160.0)
    assert bench.max_over_ranks(12.5, False) == 12.5


def test_profile_summaries_and_traffic_table_name_the_same_build(bench):
    # each committed ncu summary states the source hash it was captured on;
    # the bench's traffic table must carry the same figure for the same hash
    import re
    pdir = os.path.join(ROOT, "profiles")
    summaries = {"attn_fwd_gqa_long_step.md": ("attn_step", "gqa_long"),
                 "attn_fwd_gqa_long_refresh.md": ("attn_refresh", "gqa_long"),
                 "decode_scores_bulk_gqa_long.md": ("scores", "gqa_long")}
    for fn, key in summaries.items():
        text = open(os.path.join(pdir, fn)).read()
        sha = re.search(r"sha256 prefix ([0-9a-f]{16})", text).group(1)
        ent = bench.MEASURED_TRAFFIC[key]
        assert sha == ent["sha16"], fn
        digits = re.sub(r"[^0-9]", "", re.search(r"traffic[^|]*\|\s*([0-9,]+) B", text).group(1))
        assert int(digits) == ent["bytes"], fn
    # the one-tile and the 32-layer trajectory's summaries were captured on the same attention sources
    for fn in ("attn_fwd_single_llada_layer_step.md", "attn_fwd_traj32_step.md"):
        text = open(os.path.join(pdir, fn)).read()
        assert re.search(r"sha256 prefix ([0-9a-f]{16})", text).group(1) == \
            bench.MEASURED_TRAFFIC[("attn_step", "gqa_long")]["sha16"], fn


def test_kernel_stats_divide_each_record_by_its_launches(bench):
    """A record spans a step's layer loop (L launches back to back) or one
    scoring call; the mean is the total time over all launches of a kind."""
    class Ev:
        def __init__(self, t):
            self.t = t

        def elapsed_time(self, end):
            return end.t - self.t

    class Traj:
        attn_events = [(Ev(0.0), Ev(32 * 0.35), "step", 32), (Ev(0.0), Ev(32 * 0.37), "step", 32),
                       (Ev(0.0), Ev(32 * 3.1), "refresh", 32), (Ev(0.0), Ev(0.41), "score", 1),
                       (Ev(0.0), Ev(0.43), "score", 1)]

    ks = bench.kernel_stats(Traj())
    assert ks["step"]["count"] == 64 and ks["step"]["mean_ms"] == pytest.approx(0.36)
    assert ks["refresh"]["count"] == 32 and ks["refresh"]["mean_ms"] == pytest.approx(3.1)
    assert ks["score"]["count"] == 2 and ks["score"]["total_ms"] == pytest.approx(0.84)
