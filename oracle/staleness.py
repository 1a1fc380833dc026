"""Staleness bound of a cached step (Eq. theory-smoothness, Eq. theory-radius-bound
and their appendix form Eq. app-radius-bound) on one attention layer whose
prompt cache is the linear synthetic map of synth.staleness_model.

TEST INFRASTRUCTURE ONLY (see oracle.py).

For that map, with E(g) the stacked unit-norm response embeddings of
diameter B_e:
  ||K_p(g_t) - K_p(g_r)||_row j <= ||alpha_j||_2 ||A_K||_2 ||E(g_t) - E(g_r)||_F
                                <= ||alpha_j||_2 ||A_K||_2 B_e sqrt(D_t)       (L_C)
and for one query row o = sum_j p_j v_j (softmax p over the scores s<q, k_j>):
  o_fresh - o_cached = sum_j p'_j (v'_j - v_j) + sum_j (p'_j - p_j) v_j,
  ||p' - p||_1 <= ||x' - x||_inf   (the softmax Jacobian has inf->1 norm <= 1),
  ||x' - x||_inf <= s ||q||_2 max_j ||k'_j - k_j||_2,
so ||o_fresh - o_cached||_inf <= Gamma sqrt(D_t) with
  Gamma = B_e max_j ||alpha_j||_2 (||A_V||_2 + s max_i ||q_i||_2 ||A_K||_2 max_j ||v_j||_inf)   (L_Phi L_C B)
(v_j over the cached prompt V and the response V).  Every quantity is exact
fp64 arithmetic on the map's fp64 output.
"""
from __future__ import annotations

import math

import numpy as np

from oracle import oracle as O
from paper_2608_08086_gb300 import synth


def gamma(model: dict, q_resp, v_cache, v_resp, scale: float) -> float:
    emb = model["emb"]
    diff = emb[:, None, :] - emb[None, :, :]
    b_e = float(np.sqrt((diff ** 2).sum(-1)).max())                 # embedding diameter
    alpha_row = float(np.linalg.norm(model["alpha"], axis=1).max())
    ak = float(np.linalg.norm(model["a_k"], 2))
    av = float(np.linalg.norm(model["a_v"], 2))
    qn = float(np.linalg.norm(np.asarray(q_resp, dtype=np.float64), axis=-1).max())
    vmax = max(float(np.abs(v_cache).max()), float(np.abs(v_resp).max()))
    return b_e * alpha_row * (av + scale * qn * ak * vmax)


def curve(shape: synth.AttnShape, ds, seed: int = 0, drift: float = 0.6):
    """err(D) = ||O_cached - O_fresh||_inf over every response query and head,
    O_cached attending to K_p(g_r), O_fresh to K_p(g_t) at distance D, both
    exact (fp64 map, fp64 attention).  Returns [(D, err, Gamma sqrt(D))]."""
    B, P, G, Hq, Hkv, D = (shape.batch, shape.prompt_len, shape.resp_len, shape.n_heads, shape.n_kv_heads,
                           shape.head_dim)
    m = synth.staleness_model(shape, seed=seed, drift=drift)
    scale = 1.0 / math.sqrt(D)
    q = synth.bf16_bits_to_f64(m["q_resp"])
    kg, vg = synth.bf16_bits_to_f64(m["k_resp"]), synth.bf16_bits_to_f64(m["v_resp"])
    g_r = synth.staleness_tokens(seed, B, G)
    kc, vc = synth.staleness_prompt_cache(m, g_r, Hkv, D)
    o_cached, _ = O.attn_step(q, kc, vc, kg, vg, scale)
    gam = gamma(m, q, vc, vg, scale)
    out = []
    for d in ds:
        g_t = synth.staleness_drift(g_r, d, seed)
        kf, vf = synth.staleness_prompt_cache(m, g_t, Hkv, D)
        o_fresh, _ = O.attn_step(q, kf, vf, kg, vg, scale)
        out.append((d, float(np.abs(o_cached - o_fresh).max()), gam * math.sqrt(d)))
    return out
