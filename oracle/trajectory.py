"""Algorithm 1 (state-anchored rollback decoding) on the fp64 oracle.

TEST INFRASTRUCTURE ONLY (see oracle.py).  The rollback decoder D is replaced
by the seeded redraw of paper_2608_08086_gb300.synth (n positions per sequence
get a new token and new Q/K/V rows in every layer); everything else follows the
algorithm's order:

  step 0:  g_r <- g_0; FullForward builds the prompt cache in every layer; score.
  step t:  g <- redraw(g)                                   (stands in for D)
           D_t = d_H(g, g_r); refresh iff D_t >= K or age_t >= max_age
           refresh: FullForward per layer (prompt queries too, cache <- fresh
                    prompt K/V), g_r <- g
           else:    CachedForward per layer (response queries over [cache || response])
           score the step's logits.
``mode="eager"`` forces a refresh every step (K = 0, Eq. archer-fresh).
``decoder="closed"`` replaces the redraw by a confidence rule on the previous
step's scores (oracle.decoder_update): every position starts masked, a
changed position gets new Q/K/V rows (synth.closed_loop_rows), and the logits
plant a target token per position whose boost grows with the step
(synth.closed_loop_logits), so refresh decisions depend on scoring outputs.
"""
from __future__ import annotations

import math

import numpy as np

from oracle import oracle as O
from paper_2608_08086_gb300 import synth


def _f64(bits):
    return synth.bf16_bits_to_f64(bits)


def run(wl: synth.Workload, seed: int = 0, mode: str = "archer", steps: int | None = None,
        n_threads: int = 0, score: bool = True, decoder: str = "redraw", closed_loop: dict | None = None) -> list:
    sh = wl.shape
    B, P, G, Hq, Hkv, D = sh.batch, sh.prompt_len, sh.resp_len, sh.n_heads, sh.n_kv_heads, sh.head_dim
    N = P + G
    K = 0 if mode == "eager" else wl.radius_k
    max_age = 0 if mode == "eager" else wl.max_age
    scale = 1.0 / math.sqrt(D)
    T = wl.steps if steps is None else steps

    closed = decoder == "closed"
    cl = dict(synth.CLOSED_LOOP, **(closed_loop or {}))
    if closed:
        g = np.full((B, G), synth.MASK_TOKEN, dtype=np.int32)
    else:
        g = synth.traj_initial_tokens(wl, seed)
    layers = []
    for layer in range(wl.layers):
        x = synth.traj_layer_initial(wl, seed, layer)
        layers.append({k: _f64(v) for k, v in x.items()})

    def scores(t):
        if closed:
            z = synth.closed_loop_logits(wl, seed, t, cl["boost_per_step"])
            z = _f64(z) if wl.logits_dtype == "bf16" else z.astype(np.float64)
            return O.decode_scores(z, mask_state=(g == synth.MASK_TOKEN).astype(np.uint8), cur_tokens=g,
                                   n_threads=n_threads)
        if not score or wl.logits_rows == 0:
            return None
        z = synth.traj_logits(wl, seed, t)
        z = _f64(z) if wl.logits_dtype == "bf16" else z.astype(np.float64)
        return O.decode_scores(z, n_threads=n_threads)

    # step 0: FullForward builds the cache (Algorithm 1, first forward)
    rec = {"t": 0, "flag": np.ones(B, np.uint8), "dist": np.zeros(B, np.int32), "out": []}
    for x in layers:
        out, lse, kc, vc = O.prompt_refresh(x["q_all"], x["k_new"], x["v_new"], x["k_resp"], x["v_resp"],
                                            np.zeros_like(x["k_new"]), np.zeros_like(x["v_new"]), scale,
                                            n_threads=n_threads)
        x["k_cache"], x["v_cache"] = kc, vc
        rec["out"].append(out)
    rec["scores"] = scores(0)
    rec["g"] = g.copy()
    records = [rec]
    g_anchor = g.copy()
    age = np.zeros(B, np.int32)

    for t in range(1, T + 1):
        changed = None
        if closed:
            prev = records[-1]["scores"]
            g, changed = O.decoder_update(g, prev["max_prob"], prev["top1"], prev["cur_prob"],
                                          cl["tau_accept"], cl["tau_remask"], synth.MASK_TOKEN)
            bs, ps = np.nonzero(changed)
            for layer, x in enumerate(layers):
                rows = synth.closed_loop_rows(wl, seed, t, layer)
                x["q_all"][bs, P + ps] = _f64(rows["q"][bs, ps])
                x["k_resp"][bs, ps] = _f64(rows["k"][bs, ps])
                x["v_resp"][bs, ps] = _f64(rows["v"][bs, ps])
        else:
            pos, new = synth.traj_redraw(wl, seed, t, g)
            bidx = np.arange(B)[:, None]
            g[bidx, pos] = new
            for layer, x in enumerate(layers):
                rows = synth.traj_redraw_rows(wl, seed, t, layer)
                x["q_all"][bidx, P + pos] = _f64(rows["q"])
                x["k_resp"][bidx, pos] = _f64(rows["k"])
                x["v_resp"][bidx, pos] = _f64(rows["v"])
        dist, flag, g_anchor, age = O.should_refresh(g, g_anchor, age, K, max_age, update_anchor=True)
        rec = {"t": t, "flag": flag, "dist": dist, "out": []}
        if flag.any():
            for layer, x in enumerate(layers):
                fp = synth.traj_fresh_prompt(wl, seed, t, layer)
                x["q_all"][:, :P] = _f64(fp["q_prompt"])
                x["k_new"], x["v_new"] = _f64(fp["k_new"]), _f64(fp["v_new"])
                out, lse, kc, vc = O.prompt_refresh(x["q_all"], x["k_new"], x["v_new"], x["k_resp"],
                                                    x["v_resp"], x["k_cache"], x["v_cache"], scale, flags=flag,
                                                    n_threads=n_threads)
                x["k_cache"], x["v_cache"] = kc, vc
                rec["out"].append(out)
        else:
            for x in layers:
                out, lse = O.attn_step(x["q_all"][:, P:], x["k_cache"], x["v_cache"], x["k_resp"], x["v_resp"],
                                       scale, n_threads=n_threads)
                rec["out"].append(out)
        rec["scores"] = scores(t)
        rec["g"] = g.copy()
        rec["changed"] = changed
        records.append(rec)
    return records
