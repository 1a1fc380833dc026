"""Benchmark of the Archer denoising step on one GB300 (or N replicas).

A "step" is one pass of the whole hot path over one batch: the redraw that
stands in for the rollback decoder, the refresh rule (archer_should_refresh),
the refresh-flag read-back, attention in every layer (archer_attn_step, or
archer_prompt_refresh with the prompt-cache rewrite when the rule fires) and
decoder scoring (archer_decode_scores).  Default workload: the long-prompt GQA
trajectory (batch 16, 28 query / 4 KV heads, head_dim 128, prompt 4096,
response 512, 32 layers, 5% redraw per step, refresh every 16 steps, scoring
over a 152064-token vocabulary).

Reported on one JSON line (rank 0):
  value        denoise steps/s over K timed steps (device inputs resident in HBM)
  e2e          the same through the C ABI with every step's inputs copied from
               pinned host memory and the scores copied back
  roofline     the attention kernel: algorithmic FLOPs per launch / mean launch
               time (CUDA events on the launching stream) vs the measured bf16 peak
  speedup_vs_refresh_every_step   against the eager arm (refresh at every step)
  scoring      decode_scores GB/s vs the measured HBM copy bandwidth
  cpu_baseline the fp64 oracle on a bounded sample, on this host's cores
Every input is larger than L2 (each layer's prompt K/V alone exceeds 129 MB),
so no explicit L2 flush is done between steps.

--impl reference times the oracle (the CPU reference of this build) on bounded
samples of the same workload.  Multi-GPU (torchrun): independent replicas, one
per rank, no collective on the data path ("scaling": "weak").
"""
from __future__ import annotations

import argparse
import dataclasses
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

from paper_2608_08086_gb300 import synth  # noqa: E402

METRIC = "denoise steps/s"

# DRAM traffic per launch (dram__bytes_read.sum + dram__bytes_write.sum) from one
# ncu capture of the same launch configuration (see profiles/).  A figure is
# valid only for the kernel source it was captured on: the sha256 prefix of the
# translation unit is checked at run time and the figure dropped on mismatch.
MEASURED_TRAFFIC = {
    # (kernel, workload): DRAM bytes read + written per launch from one ncu capture
    # (dram__bytes_read.sum + dram__bytes_write.sum), valid only while the kernel's
    # sources hash to sha16 (sha256 over the listed files, first 16 hex digits).
    ("attn_step", "gqa_long"): {"bytes": 209797120 + 37160448, "sha16": "bba83f495a267f1c",
                                "sources": ["attention_kernels.cuh", "attention_step.cu", "archer_device.cuh",
                                            "tmem_ldst.cuh"]},
    ("attn_refresh", "gqa_long"): {"bytes": 812074496 + 624359680, "sha16": "8dfd63cb241930e0",
                                   "sources": ["attention_kernels.cuh", "attention_rewrite.cu", "archer_device.cuh",
                                               "tmem_ldst.cuh"]},
    ("scores", "gqa_long"): {"bytes": 2491648000 + 4957440, "sha16": "a5463d9160dc1f66",
                             "sources": ["decode_scores.cu", "archer_device.cuh"]},
}


def _source_sha(files):
    import hashlib
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, "paper_2608_08086_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def measured_traffic(kernel, workload):
    ent = MEASURED_TRAFFIC.get((kernel, workload))
    if not ent:
        return None
    try:
        return ent["bytes"] if _source_sha(ent["sources"]) == ent["sha16"] else None
    except OSError:
        return None


PEAKS_FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return p, "measured"
    except (OSError, ValueError):
        return PEAKS_FALLBACK, "fallback"


# ---------------------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi clocks and throttle reasons, sampled every 200 ms."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        out = {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        if self.proc is None:
            return out
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return out
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        out["samples"] = len(rows)
        out["sm_mhz"] = statistics.median(sm) if sm else None
        out["sm_max_mhz"] = max(float(r[2]) for r in rows if r[2].replace(".", "").isdigit()) if sm else None
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        reasons = set()
        for r in rows:
            for name, v in zip(names, r[5:9]):
                if v.lower() == "active":
                    reasons.add(name)
        out["reasons"] = sorted(reasons)
        return out


# ---------------------------------------------------------------------------- timing helpers

def barrier(dist_on, device="cuda"):
    if dist_on:
        torch.distributed.barrier()
    if device == "cuda":
        torch.cuda.synchronize()


def max_over_ranks(x: float, dist_on: bool, device="cuda") -> float:
    """The slowest rank's time: the job's time (replicas run in lock-step
    between barriers)."""
    if not dist_on:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(world: int, steps: int, ms: float) -> float:
    """Steps per second of the whole job: every rank (one replica per GPU)
    completes `steps` steps in the slowest rank's `ms`."""
    return world * steps / (ms / 1e3)


def run_arm(wl, mode, steps, warmup, dist_on, time_attention=False, seed=0):
    from paper_2608_08086_gb300.trajectory import DeviceTrajectory
    tr = DeviceTrajectory(wl, seed=seed, mode=mode, source="device", max_steps=warmup + steps + 1)
    tr.build()
    for _ in range(warmup):
        tr.step()
    barrier(dist_on)
    tr.time_attention = time_attention
    tr.attn_events = []
    refresh_before = tr.n_refresh_steps
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.nvtx.range_push(f"timed-{mode}")
    start.record()
    for _ in range(steps):
        tr.step()
    end.record()
    torch.cuda.nvtx.range_pop()
    barrier(dist_on)
    ms = start.elapsed_time(end)
    info = {"ms": ms, "refresh_steps": tr.n_refresh_steps - refresh_before, "traj": tr}
    return info


def kernel_only(args, wl):
    """A few launches of one kernel on the workload's full-size tensors (for
    profiler captures): attn_step | attn_refresh | scores."""
    from paper_2608_08086_gb300 import archer as A
    sh = wl.shape
    B, P, G, Hq, Hkv, D = sh.batch, sh.prompt_len, sh.resp_len, sh.n_heads, sh.n_kv_heads, sh.head_dim
    dev = torch.device("cuda")
    if args.kernel_only.startswith("attn"):
        d = synth.device_attn_inputs(sh, dev, seed=0)
        shape = A.make_shape(B, P, G, Hq, Hkv, D)
        if args.kernel_only == "attn_step":
            q = d["q_all"][:, P:].contiguous()
            out = torch.empty(B, G, Hq, D, dtype=torch.bfloat16, device=dev)
            fn = lambda: A.archer_attn_step(shape, q, d["k_cache"], d["v_cache"], d["k_resp"], d["v_resp"], out)  # noqa: E731
        else:
            # the cache is a buffer of its own, as in the trajectory: the launch rewrites it
            out = torch.empty(B, P + G, Hq, D, dtype=torch.bfloat16, device=dev)
            fn = lambda: A.archer_prompt_refresh(shape, d["q_all"], d["k_prompt"], d["v_prompt"], d["k_resp"],  # noqa: E731
                                                 d["v_resp"], out, None, d["k_cache"], d["v_cache"])
    else:
        rows = wl.logits_rows
        z = synth.device_logits(rows, wl.vocab, dev, seed=0, std=wl.logits_std, boost_max=wl.logits_boost)
        mp = torch.empty(rows, dtype=torch.float32, device=dev)
        t1 = torch.empty(rows, dtype=torch.int32, device=dev)
        mg = torch.empty(rows, dtype=torch.float32, device=dev)
        fn = lambda: A.archer_decode_scores(z, mp, t1, mg)  # noqa: E731
    for _ in range(args.warmup):
        fn()
    torch.cuda.synchronize()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    start.record()
    for _ in range(args.launches):
        fn()
    end.record()
    torch.cuda.synchronize()
    A.archer_check_device()
    print(json.dumps({"kernel_only": args.kernel_only, "workload": wl.name, "launches": args.launches,
                      "mean_ms": start.elapsed_time(end) / args.launches}), flush=True)
    return 0


def _time_graph(fn, runs):
    """Mean duration in us of fn's launches replayed back to back from one CUDA
    graph of `runs` launches: the device-side cost, free of the host's launch
    rate (which bounds plain back-to-back launches of layers this small)."""
    g = torch.cuda.CUDAGraph()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        fn()
    torch.cuda.current_stream().wait_stream(side)
    with torch.cuda.graph(g):
        for _ in range(runs):
            fn()
    g.replay()
    torch.cuda.synchronize()
    s, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s.record()
    g.replay()
    e.record()
    e.synchronize()
    del g
    return s.elapsed_time(e) * 1e3 / runs


def _time_launches(fn, runs, flush=None):
    """Median (cold: L2 flushed before each launch) and mean back-to-back
    duration in us of fn's launches, CUDA events on the current stream."""
    cold = []
    for _ in range(runs):
        if flush is not None:
            flush.add_(1)
        s, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s.record()
        fn()
        e.record()
        e.synchronize()
        cold.append(s.elapsed_time(e) * 1e3)
    s, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s.record()
    for _ in range(runs):
        fn()
    e.record()
    e.synchronize()
    return statistics.median(cold), s.elapsed_time(e) * 1e3 / runs


def _attn_pair(sh, dev, runs, flush):
    """Cached step and refresh of one layer of shape sh: times and TFLOP/s."""
    from paper_2608_08086_gb300 import archer as A
    B, P, G, Hq, Hkv, D = sh.batch, sh.prompt_len, sh.resp_len, sh.n_heads, sh.n_kv_heads, sh.head_dim
    d = synth.device_attn_inputs(sh, dev, seed=0)
    shape = A.make_shape(B, P, G, Hq, Hkv, D)
    q = d["q_all"][:, P:].contiguous()
    out_g = torch.empty(B, G, Hq, D, dtype=torch.bfloat16, device=dev)
    out_n = torch.empty(B, P + G, Hq, D, dtype=torch.bfloat16, device=dev)
    step = lambda: A.archer_attn_step(shape, q, d["k_cache"], d["v_cache"], d["k_resp"], d["v_resp"], out_g)  # noqa: E731
    refresh = lambda: A.archer_prompt_refresh(shape, d["q_all"], d["k_prompt"], d["v_prompt"], d["k_resp"],  # noqa: E731
                                              d["v_resp"], out_n, None, d["k_prompt"], d["v_prompt"])
    for _ in range(3):
        step()
        refresh()
    torch.cuda.synchronize()
    N = P + G
    res = {}
    for name, fn, M in (("step", step, G), ("refresh", refresh, N)):
        cold, b2b = _time_launches(fn, runs, flush)
        gr = _time_graph(fn, runs)
        fl = 4.0 * B * Hq * M * N * D
        res[name] = {"cold_us": cold, "b2b_us": b2b, "graph_us": gr, "gflop": fl / 1e9, "tflops_cold": fl / cold / 1e6,
                     "tflops_b2b": fl / b2b / 1e6, "tflops_graph": fl / gr / 1e6}
    A.archer_check_device()
    res["refresh_over_step"] = res["refresh"]["cold_us"] / res["step"]["cold_us"]
    res["ideal_ratio_N_over_G"] = N / G
    return res


def per_config(runs, pk, pk_kind):
    """Per-configuration measurements: the LLaDA-shaped layer (B1, 32 = 32
    heads, D128, P512, G256; cached step next to its 768-query refresh),
    decoder scoring on [4 x 256 x 126464] bf16, and the prompt-length sweep
    G = 256, P = 128 ... 2048 with LLaDA heads (cached step vs refresh of one
    layer).  "cold" launches follow a 256 MB L2-flushing write; "b2b" is back
    to back from the host; "graph" is back to back from one captured CUDA
    graph (the device-side cost of a layer in a chain).  These kernels are
    timed alone, so their fractions are of the burst peaks."""
    from paper_2608_08086_gb300 import archer as A
    dev = torch.device("cuda")
    flush = torch.zeros(64 << 20, dtype=torch.float32, device=dev)     # 256 MB > L2
    peak_tf = pk["bf16_tflops"]

    def attn(sh):
        r = _attn_pair(sh, dev, runs, flush)
        for k in ("step", "refresh"):
            r[k]["frac_graph"] = r[k]["tflops_graph"] / peak_tf
            r[k]["frac_cold"] = r[k]["tflops_cold"] / peak_tf
        r["refresh_over_step_graph"] = r["refresh"]["graph_us"] / r["step"]["graph_us"]
        return r

    out = {"peak_tflops": peak_tf, "peak_gbs": pk["hbm_gbs"], "peak_kind": f"burst ({pk_kind})", "runs": runs}
    wl = synth.WORKLOADS["llada_layer"]
    out["llada_layer"] = {"shape": dataclasses.asdict(wl.shape), **attn(wl.shape)}
    wl = synth.WORKLOADS["scoring"]
    rows = wl.logits_rows
    z = synth.device_logits(rows, wl.vocab, dev, seed=0, std=wl.logits_std, boost_max=wl.logits_boost)
    mp = torch.empty(rows, dtype=torch.float32, device=dev)
    t1 = torch.empty(rows, dtype=torch.int32, device=dev)
    mg = torch.empty(rows, dtype=torch.float32, device=dev)
    ws = A.scores_workspace(rows, wl.vocab, dev)
    fn = lambda: A.archer_decode_scores(z, mp, t1, mg, workspace=ws)  # noqa: E731
    for _ in range(3):
        fn()
    cold, b2b = _time_launches(fn, runs, flush)
    gr = _time_graph(fn, runs)
    nbytes = rows * wl.vocab * 2
    out["scoring"] = {"rows": rows, "vocab": wl.vocab, "bytes": nbytes, "cold_us": cold, "b2b_us": b2b,
                      "graph_us": gr, "gbs_cold": nbytes / cold / 1e3, "gbs_graph": nbytes / gr / 1e3,
                      "frac_cold": nbytes / cold / 1e3 / pk["hbm_gbs"], "frac_graph": nbytes / gr / 1e3 / pk["hbm_gbs"]}
    del z, mp, t1, mg, ws
    sweep_pts = []
    for P in (128, 256, 512, 1024, 2048):
        sh = synth.AttnShape(1, P, 256, 32, 32, 128)
        sweep_pts.append({"P": P, "G": 256, **attn(sh)})
    out["prompt_sweep"] = sweep_pts
    A.archer_check_device()
    del flush
    torch.cuda.empty_cache()
    return out


def sweep(args):
    """The per-configuration measurements of per_config, one JSON line each."""
    pk, pk_kind = peaks()
    res = per_config(max(args.launches, 20), pk, pk_kind)
    print(json.dumps({"sweep": "llada_layer", "runs": res["runs"], **res["llada_layer"]}), flush=True)
    print(json.dumps({"sweep": "scoring", **res["scoring"], "peak_gbs": res["peak_gbs"],
                      "peak_kind": res["peak_kind"]}), flush=True)
    for pt in res["prompt_sweep"]:
        print(json.dumps({"sweep": "prompt_len", "runs": res["runs"], **pt}), flush=True)
    return 0


def compact_configs(res):
    """The per-configuration results as they go on the bench line: per
    attention layer the graph-replayed and cold times (us), TFLOP/s and
    fraction of the burst bf16 peak, per scoring launch GB/s and fraction of
    the HBM copy peak."""
    def attn(r):
        return {k: {"graph_us": round(r[k]["graph_us"], 2), "cold_us": round(r[k]["cold_us"], 2),
                    "gflop": round(r[k]["gflop"], 3), "tflops_graph": round(r[k]["tflops_graph"], 1),
                    "frac_graph": round(r[k]["frac_graph"], 4), "tflops_cold": round(r[k]["tflops_cold"], 1)}
                for k in ("step", "refresh")} | {"refresh_over_step_graph": round(r["refresh_over_step_graph"], 3),
                                                 "ideal_ratio_N_over_G": r["ideal_ratio_N_over_G"]}
    sc = res["scoring"]
    return {"peak_tflops": res["peak_tflops"], "peak_gbs": res["peak_gbs"], "peak_kind": res["peak_kind"],
            "timing": "graph = mean of launches replayed from one CUDA graph; cold = median single launch after "
                      "a 256 MB L2-flushing write",
            "llada_layer": {"shape": "B1, 32/32 heads, D128, P512, G256", **attn(res["llada_layer"])},
            "scoring": {"shape": "bf16 [4 x 256 x 126464]", "bytes": sc["bytes"],
                        "graph_us": round(sc["graph_us"], 2), "cold_us": round(sc["cold_us"], 2),
                        "gbs_graph": round(sc["gbs_graph"], 1), "frac_graph": round(sc["frac_graph"], 4),
                        "gbs_cold": round(sc["gbs_cold"], 1), "frac_cold": round(sc["frac_cold"], 4)},
            "prompt_sweep": [{"P": pt["P"], "G": pt["G"], **attn(pt)} for pt in res["prompt_sweep"]]}


def staleness(args):
    """The staleness curve of a cached step (Eq. theory-radius-bound) on a
    LLaDA-shaped layer (B1, 32 heads, D128, P512, G256) whose prompt cache is
    the linear synthetic map of synth.staleness_model: the CUDA cached step
    against K_p(g_r) and against K_p(g_t) at Hamming distance D (caches in
    bf16), err = max |O_cached - O_fresh|, and the bound Gamma sqrt(D) of that
    map (one JSON line per D)."""
    from paper_2608_08086_gb300 import archer as A
    shape = synth.AttnShape(1, 512, 256, 32, 32, 128)
    B, P, G, Hq, Hkv, D = 1, 512, 256, 32, 32, 128
    m = synth.staleness_model(shape, seed=0)
    scale = 1.0 / math.sqrt(D)
    dev = torch.device("cuda")

    def dev_bits(bits):
        return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(dev)

    g_r = synth.staleness_tokens(0, B, G)
    kc, vc = synth.staleness_prompt_cache(m, g_r, Hkv, D)
    kc_b, vc_b = synth.to_bf16_bits(kc), synth.to_bf16_bits(vc)
    q, kg, vg = dev_bits(m["q_resp"]), dev_bits(m["k_resp"]), dev_bits(m["v_resp"])
    sh = A.make_shape(B, P, G, Hq, Hkv, D)
    # Gamma = B_e max_j ||alpha_j|| (||A_V|| + s max ||q|| ||A_K|| max |v|)  (L_Phi L_C B)
    emb = m["emb"]
    b_e = float(np.sqrt(((emb[:, None] - emb[None]) ** 2).sum(-1)).max())
    f64 = synth.bf16_bits_to_f64
    qn = float(np.linalg.norm(f64(m["q_resp"]), axis=-1).max())
    vmax = max(float(np.abs(f64(vc_b)).max()), float(np.abs(f64(m["v_resp"])).max()))
    gam = b_e * float(np.linalg.norm(m["alpha"], axis=1).max()) * (
        float(np.linalg.norm(m["a_v"], 2)) + scale * qn * float(np.linalg.norm(m["a_k"], 2)) * vmax)

    def run(kb, vb):
        out = torch.empty(B, G, Hq, D, dtype=torch.bfloat16, device=dev)
        A.archer_attn_step(sh, q, dev_bits(kb), dev_bits(vb), kg, vg, out)
        return out.float()

    o_cached = run(kc_b, vc_b)
    for d in (0, 1, 2, 4, 8, 16, 32, 64, 128, 256):
        kf, vf = synth.staleness_prompt_cache(m, synth.staleness_drift(g_r, d, 0), Hkv, D)
        err = float((run(synth.to_bf16_bits(kf), synth.to_bf16_bits(vf)) - o_cached).abs().max())
        print(json.dumps({"staleness": "llada_layer", "D_t": d, "err_inf": err, "gamma_sqrt_d": gam * math.sqrt(d),
                          "err_over_sqrt_d": err / math.sqrt(d) if d else 0.0, "gamma": gam}), flush=True)
    A.archer_check_device()
    return 0


def kernel_stats(tr):
    """Mean durations (ms) and counts of the attention / scoring launches:
    each record spans `launches` launches of one kind back to back (a step's
    layer loop, or one scoring call), and the mean is total time / launches."""
    by = {}
    for s, e, kind, n in tr.attn_events:
        t = by.setdefault(kind, [0.0, 0])
        t[0] += s.elapsed_time(e)
        t[1] += n
    return {k: {"count": n, "mean_ms": ms / n, "total_ms": ms} for k, (ms, n) in by.items()}


# ---------------------------------------------------------------------------- e2e

def run_e2e(wl, steps, warmup, dist_on, seed=0):
    """The same step through the C ABI with HOST inputs: every step copies its
    inputs (token updates, redrawn Q/K/V rows of every layer, the step's logits,
    and at a refresh the fresh prompt Q/K/V of every layer) from pinned host
    memory and reads the scores back.  The per-step uploads are double-buffered
    on a copy stream (step t+2's inputs are uploaded while step t computes);
    a refresh step's prompt uploads start once the rule has fired, layer by
    layer on a second copy stream, each layer's refresh waiting for its own.
    The timed region starts before the first upload and issues exactly the
    uploads of the timed steps."""
    from paper_2608_08086_gb300.trajectory import DeviceTrajectory
    tr = DeviceTrajectory(wl, seed=seed, mode="archer", source="device", max_steps=warmup + steps + 2)
    sh = wl.shape
    B, P, G, L = sh.batch, sh.prompt_len, sh.resp_len, tr.L
    copy_stream = torch.cuda.Stream()
    nb = lambda t: t.numel() * t.element_size()  # noqa: E731
    # host sources (pinned): one step's redraw rows, the logits, one layer's fresh prompt
    h_rows = {c: tr.pool[c][0].cpu().pin_memory() for c in ("q", "k", "v")}
    h_logits = tr.logits.cpu().pin_memory()
    h_plan = [(p.cpu().pin_memory(), v.cpu().pin_memory()) for p, v in tr.plan]
    h_q_prompt = tr.q_all[0][:, :P].contiguous().cpu().pin_memory()
    h_k_new = tr.k_new[0].cpu().pin_memory()
    h_v_new = tr.v_new[0].cpu().pin_memory()
    h_scores = torch.empty(3, B * G, dtype=torch.float32).pin_memory()
    # device staging, two sets
    d_rows = [{c: torch.empty_like(tr.pool[c][0]) for c in ("q", "k", "v")} for _ in range(2)]
    d_logits = [tr.logits, torch.empty_like(tr.logits)]
    d_plan = [(torch.empty_like(tr.plan[0][0]), torch.empty_like(tr.plan[0][1])) for _ in range(2)]
    ready = [torch.cuda.Event() for _ in range(2)]
    consumed = [torch.cuda.Event() for _ in range(2)]
    for e in consumed:
        e.record()

    def upload(t):
        slot = t & 1
        hp, hn = h_plan[(t - 1) % len(h_plan)]
        with torch.cuda.stream(copy_stream):
            copy_stream.wait_event(consumed[slot])
            d_plan[slot][0].copy_(hp, non_blocking=True)
            d_plan[slot][1].copy_(hn, non_blocking=True)
            for c in ("q", "k", "v"):
                d_rows[slot][c].copy_(h_rows[c], non_blocking=True)
            d_logits[slot].copy_(h_logits, non_blocking=True)
            ready[slot].record(copy_stream)

    def stage_redraw(t):
        slot = t & 1
        torch.cuda.current_stream().wait_event(ready[slot])
        pos, new = d_plan[slot]
        bidx = torch.arange(B, device=tr.device)[:, None]
        tr.g[bidx, pos] = new
        tr._scatter(d_rows[slot]["q"], d_rows[slot]["k"], d_rows[slot]["v"], pos)
        tr.logits = d_logits[slot]

    fresh_stream = torch.cuda.Stream()
    layer_ready = [torch.cuda.Event() for _ in range(L)]
    tr.layer_ready = layer_ready

    def stage_fresh(t):
        # Per-layer uploads on their own stream: layer l's refresh waits only for
        # its own prompt Q/K/V, so later layers' copies overlap earlier layers' work.
        # The prompt rows of q_all ([B, N, Hq, D]) are contiguous per sequence:
        # one host-to-device copy each, done by the copy engine (a strided
        # destination would need a device kernel, competing with the attention
        # for SMs).
        here = torch.cuda.Event()
        here.record()
        with torch.cuda.stream(fresh_stream):
            fresh_stream.wait_event(here)
            for layer in range(L):
                for b in range(B):
                    tr.q_all[layer][b, :P].copy_(h_q_prompt[b], non_blocking=True)
                tr.k_new[layer].copy_(h_k_new, non_blocking=True)
                tr.v_new[layer].copy_(h_v_new, non_blocking=True)
                layer_ready[layer].record(fresh_stream)

    tr._stage_redraw = stage_redraw
    tr._stage_fresh_prompt = stage_fresh
    per_step_in = nb(h_plan[0][0]) + nb(h_plan[0][1]) + sum(nb(h) for h in h_rows.values()) + nb(h_logits)
    per_refresh_in = L * (nb(h_q_prompt) + nb(h_k_new) + nb(h_v_new))

    def run_steps(first, count):
        upload(first)
        if count > 1:
            upload(first + 1)
        for i in range(count):
            t = first + i
            tr.step()
            h_scores[0].copy_(tr.max_prob, non_blocking=True)
            h_scores[1].copy_(tr.top1.view(torch.float32), non_blocking=True)
            h_scores[2].copy_(tr.margin, non_blocking=True)
            consumed[t & 1].record()
            if i + 2 < count:
                upload(t + 2)

    tr.build()
    run_steps(1, warmup)
    barrier(dist_on)
    r0 = tr.n_refresh_steps
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    start.record()
    run_steps(warmup + 1, steps)
    end.record()
    barrier(dist_on)
    ms = start.elapsed_time(end)
    n_ref = tr.n_refresh_steps - r0
    h2d = (steps * per_step_in + n_ref * per_refresh_in) / steps
    d2h = B + 3 * B * G * 4      # the refresh flags and the three score vectors
    del tr
    torch.cuda.empty_cache()
    return {"ms": ms, "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h), "overlap": "copy streams (per-step double buffer; per-layer refresh uploads)"}


# ---------------------------------------------------------------------------- oracle (CPU)

def refresh_fraction(wl, seed=0):
    """Share of (sequence, step) pairs of the workload's denoising steps
    1..T that refresh, from the oracle's rule (Eq. archer-distance, the age
    cap) over the workload's own seeded redraws."""
    from oracle import oracle as O
    from paper_2608_08086_gb300 import synth
    B = wl.shape.batch
    if wl.steps < 1 or B < 1:
        return 0.0
    g = synth.traj_initial_tokens(wl, seed)
    anchor, age = g.copy(), np.zeros(B, np.int32)
    fired = 0
    for t in range(1, wl.steps + 1):
        pos, new = synth.traj_redraw(wl, seed, t, g)
        g[np.arange(B)[:, None], pos] = new
        _, flag, anchor, age = O.should_refresh(g, anchor, age, wl.radius_k, wl.max_age)
        fired += int(flag.sum())
    return fired / (B * wl.steps)


def oracle_sample_step(wl, n_pairs=None, score_rows=8, seed=0):
    """One bounded sample of a step on the fp64 oracle, extrapolated to the full
    step: cached attention of `n_pairs` (sequence, head) pairs of one layer, one
    refresh pair, and scoring of `score_rows` rows; scaled by the workload's
    pair, layer and row counts and its refresh fraction.  Returns
    (seconds per full step, sample description, threads)."""
    from oracle import oracle as O
    sh = wl.shape
    B, P, G, Hq, Hkv, D = sh.batch, sh.prompt_len, sh.resp_len, sh.n_heads, sh.n_kv_heads, sh.head_dim
    threads = O.hardware_threads()
    n_pairs = n_pairs or max(1, threads)
    rng = np.random.default_rng(seed)
    std = 1.0 / math.sqrt(D)
    q = rng.standard_normal((1, G, n_pairs, D)) * std
    kc = rng.standard_normal((1, P, n_pairs, D)) * std
    vc = rng.standard_normal((1, P, n_pairs, D)) * std
    kg = rng.standard_normal((1, G, n_pairs, D)) * std
    vg = rng.standard_normal((1, G, n_pairs, D)) * std
    t0 = time.perf_counter()
    O.attention(q, kc, vc, kg, vg, 1.0 / math.sqrt(D), n_threads=threads)      # n_pairs independent heads
    t_cached_pairs = time.perf_counter() - t0
    # refresh costs N/G times a cached pair (N queries instead of G)
    t_refresh_pair = t_cached_pairs / n_pairs * (P + G) / G
    t_score = 0.0
    if wl.logits_rows:
        z = rng.standard_normal((score_rows, wl.vocab)) * wl.logits_std
        t0 = time.perf_counter()
        O.decode_scores(z, n_threads=threads)
        t_score = (time.perf_counter() - t0) / score_rows * wl.logits_rows
    pairs = B * Hq
    q_k = refresh_fraction(wl, seed)
    per_layer = (1 - q_k) * t_cached_pairs / n_pairs * pairs + q_k * t_refresh_pair * pairs
    step_s = wl.layers * per_layer + t_score
    sample = (f"{n_pairs} (sequence, head) pairs of one cached layer ({G} queries x {P + G} keys, D={D}) and "
              f"{score_rows} scoring rows of {wl.vocab}, extrapolated to {pairs} pairs x {wl.layers} layers with "
              f"refresh fraction {q_k:.3f} and {wl.logits_rows} rows")
    return step_s, sample, threads


def config_of(wl, world):
    """The workload's configuration as both arms print it."""
    return {"workload": wl.name, "batch": wl.shape.batch, "prompt_len": wl.shape.prompt_len,
            "resp_len": wl.shape.resp_len, "n_heads": wl.shape.n_heads, "n_kv_heads": wl.shape.n_kv_heads,
            "head_dim": wl.shape.head_dim, "layers": wl.layers, "vocab": wl.vocab,
            "redraws_per_step": wl.redraws_per_step, "max_age": wl.max_age,
            "radius_k": None if wl.radius_k >= synth.K_INFINITE else wl.radius_k,
            "parallelism": f"replicas{world}" if world > 1 else "single",
            "l2": "no flush: inputs larger than L2 (prompt K/V of one layer > 129 MB)"}


def reference_arm(args, wl):
    """The oracle timed as it stands, each step the same bounded sample as the
    default run's cpu_baseline (one (sequence, head) pair per host thread,
    8 scoring rows), extrapolated to the whole step."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    for _ in range(args.warmup):
        oracle_sample_step(wl)
    times = []
    sample = ""
    threads = 0
    for _ in range(args.steps):
        s, sample, threads = oracle_sample_step(wl)
        times.append(s)
    step_s = statistics.median(times)
    value = 1.0 / step_s
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "steps/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": step_s * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": config_of(wl, 1),
            "cpu_baseline": {"kind": "oracle", "value": value, "unit": "steps/s", "cores": threads,
                             "sample": sample + " per step (extrapolated)"},
            "e2e": {"value": value, "unit": "steps/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ---------------------------------------------------------------------------- main

def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="gqa_long", choices=["gqa_long", "traj32", "llada_layer"])
    ap.add_argument("--eager-steps", type=int, default=8)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--no-secondary", action="store_true")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the per-configuration measurements (LLaDA layer, scoring, prompt sweep)")
    ap.add_argument("--kernel-only", choices=["attn_step", "attn_refresh", "scores"], default=None,
                    help="run only a few launches of one kernel (for profiler captures)")
    ap.add_argument("--launches", type=int, default=3)
    ap.add_argument("--staleness", action="store_true",
                    help="staleness curve of a cached step against the Hamming distance (Eq. theory-radius-bound)")
    ap.add_argument("--sweep", action="store_true",
                    help="per-configuration measurements (LLaDA layer, scoring, prompt-length sweep)")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    if args.workload == "llada_layer" and args.kernel_only not in ("attn_step", "attn_refresh"):
        ap.error("llada_layer is a single attention layer: use it with --kernel-only attn_step|attn_refresh")
    wl = synth.WORKLOADS[args.workload]

    if args.impl == "reference":
        return reference_arm(args, wl)
    if args.kernel_only or args.sweep or args.staleness:
        torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
        from paper_2608_08086_gb300 import build as Bld
        Bld.build()
        if args.staleness:
            return staleness(args)
        return sweep(args) if args.sweep else kernel_only(args, wl)

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist_on = world > 1
    torch.cuda.set_device(local)
    if dist_on:
        torch.distributed.init_process_group("nccl", device_id=torch.device("cuda", local))

    from paper_2608_08086_gb300 import build as B
    B.build()
    from paper_2608_08086_gb300 import archer as A  # noqa: F401  (fails loudly without libarcher)

    pk, pk_kind = peaks()
    clocks = ClockSampler(local)

    # ---- the Archer arm (timed region = K steps): one step graph per step,
    # the refresh branch taken on the device (no host synchronisation)
    clocks.start()
    arm = run_arm(wl, "graph", args.steps, args.warmup, dist_on)
    clk = clocks.stop()
    ms = max_over_ranks(arm["ms"], dist_on)
    value = whole_job_rate(world, args.steps, ms)
    n_ref = arm["refresh_steps"]
    del arm
    torch.cuda.empty_cache()
    # ---- the same steps driven from the host (flags read back each step), with
    # CUDA events around each step's layer loop (its L attention launches back
    # to back, as in the graph step: an event between two launches would keep
    # the second from starting while the first ends) and around every scoring
    # call: the per-kernel durations of the roofline
    arm = run_arm(wl, "archer", args.steps, args.warmup, dist_on, time_attention=True)
    tr = arm["traj"]
    host_value = whole_job_rate(world, args.steps, max_over_ranks(arm["ms"], dist_on))
    ks = kernel_stats(tr)
    L = tr.L
    # per step: 3 row scatters + rule + refresh condition + L attention + scoring (2);
    # a refresh rewrites the prompt cache inside its attention launch
    launches = args.steps * (3 + 2 + L + (2 if tr.score else 0))
    flops_step_launch = 4.0 * tr.B * tr.Hq * tr.G * tr.N * tr.D
    flops_refresh_launch = 4.0 * tr.B * tr.Hq * tr.N * tr.N * tr.D
    att = {}
    tot_flops, tot_ms = 0.0, 0.0
    for kind, fl in (("step", flops_step_launch), ("refresh", flops_refresh_launch)):
        if kind in ks:
            k = ks[kind]
            att[kind] = {"launches": k["count"], "mean_ms": k["mean_ms"], "tflops": fl / (k["mean_ms"] * 1e9),
                         "traffic": measured_traffic(f"attn_{kind}", wl.name)}
            tot_flops += fl * k["count"]
            tot_ms += k["total_ms"]
    peak_tf = pk["bf16_tflops_sustained"]
    # roofline of the dominant kernel: its cached-step launches (one FLOP count)
    achieved = att["step"]["tflops"] if "step" in att else (tot_flops / (tot_ms * 1e9) if tot_ms else 0.0)
    scoring = None
    if "score" in ks:
        sbytes = tr.B * tr.G * wl.vocab * (2 if wl.logits_dtype == "bf16" else 4)
        gbs = sbytes / (ks["score"]["mean_ms"] * 1e6)
        scoring = {"mean_ms": ks["score"]["mean_ms"], "gbs": gbs, "peak_gbs": pk["hbm_gbs"],
                   "frac": gbs / pk["hbm_gbs"], "bytes_per_launch": sbytes,
                   "traffic": measured_traffic("scores", wl.name)}
    del arm, tr
    torch.cuda.empty_cache()

    # ---- the eager arm: refresh every step (one graph per step, like the Archer arm)
    eager = run_arm(wl, "eager-graph", args.eager_steps, 3, dist_on)
    eager_ms = max_over_ranks(eager["ms"], dist_on)
    eager_value = whole_job_rate(world, args.eager_steps, eager_ms)
    del eager
    torch.cuda.empty_cache()

    # ---- e2e through host buffers
    e2e = None
    if not args.no_e2e:
        e = run_e2e(wl, args.steps, args.warmup, dist_on)
        e_ms = max_over_ranks(e["ms"], dist_on)
        e2e = {"value": whole_job_rate(world, args.steps, e_ms), "unit": "steps/s",
               "h2d_bytes_per_step": e["h2d_bytes_per_step"], "d2h_bytes_per_step": e["d2h_bytes_per_step"]}

    # ---- a second trajectory workload (32 layers, B 8, P 1024, G 512, rule K=65 / age 8)
    secondary = None
    if not args.no_secondary and args.workload != "traj32":
        wl2 = synth.WORKLOADS["traj32"]
        n2 = min(args.steps, 30)
        a2 = run_arm(wl2, "graph", n2, 3, dist_on)
        v2 = whole_job_rate(world, n2, max_over_ranks(a2["ms"], dist_on))
        r2 = a2["refresh_steps"]
        del a2
        h2 = run_arm(wl2, "archer", n2, 3, dist_on, time_attention=True)
        ks2 = kernel_stats(h2["traj"])
        vh2 = whole_job_rate(world, n2, max_over_ranks(h2["ms"], dist_on))
        t2 = h2["traj"]
        e2 = run_arm(wl2, "eager-graph", args.eager_steps, 3, dist_on)
        ve2 = whole_job_rate(world, args.eager_steps, max_over_ranks(e2["ms"], dist_on))
        fl2 = 4.0 * t2.B * t2.Hq * t2.G * t2.N * t2.D
        secondary = {"workload": wl2.name, "steps_per_s": v2, "host_driven_steps_per_s": vh2,
                     "eager_steps_per_s": ve2, "speedup_vs_refresh_every_step": v2 / ve2, "refresh_steps": r2,
                     "step_attention_tflops": fl2 / (ks2["step"]["mean_ms"] * 1e9) if "step" in ks2 else None}
        del h2, e2, t2
        torch.cuda.empty_cache()

    # ---- the single-layer configurations: the LLaDA-shaped layer, scoring on
    # [4 x 256 x 126464], the prompt-length sweep (each GPU measures its own)
    configs = None
    if not args.no_configs:
        configs = compact_configs(per_config(20, pk, pk_kind))

    # ---- CPU baseline: the oracle on a bounded sample (rank 0, N = 1)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        s, sample, threads = oracle_sample_step(wl)
        cpu = {"value": 1.0 / s, "unit": "steps/s", "cores": threads, "kind": "oracle", "sample": sample}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "steps/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": config_of(wl, world),
            "refresh_steps_timed": n_ref,
            "step": "CUDA graph per step, refresh branch on the device",
            "host_driven_steps_per_s": host_value,
            "speedup_vs_refresh_every_step": value / eager_value,
            "eager_steps_per_s": eager_value,
            "attention": att,
            "roofline": {"bound": "tensor", "kernel": "attn_fwd_persist_kernel<128, 0, 0> (persistent two-tile; no rewrite, no single-tile tail)", "launches": "cached step",
                         "timing": "CUDA events around each cached step's layer loop (host-driven arm), / its launches",
                         "flops_per_launch": flops_step_launch, "achieved": achieved, "peak": peak_tf,
                         "unit": "TFLOP/s", "frac": achieved / peak_tf,
                         "traffic": measured_traffic("attn_step", wl.name),
                         "peak_kind": f"bf16_tflops_sustained ({pk_kind}; the kernel runs inside a long step)"},
            "scoring": scoring,
            "e2e": e2e,
            "gpu_launches": launches,
            "clocks": {"sm_mhz": clk["sm_mhz"], "sm_max_mhz": clk["sm_max_mhz"], "reasons": clk["reasons"]},
            "secondary": secondary,
            "configs": configs,
            "cpu_baseline": cpu,
        }
        print(json.dumps(line), flush=True)
    if dist_on:
        torch.distributed.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
