"""Seeded synthetic inputs for the Archer denoising step.

This module is the only code shared by the CUDA path's callers (tests, bench)
and the fp64 oracle.  It holds none of the method's arithmetic: only a
counter-based random number generator, normal deviates, rounding of fp64
draws to bf16 / fp32, and the workload recipes (shapes and value
distributions) that stand in for the paper's code-generation workloads
(MBPP / HumanEval / LiveCodeBench prompts with a revisable response; the
datasets themselves are not used).

Generator
---------
* SplitMix64 (Steele, Lea and Flood, "Fast splittable pseudorandom number
  generators", OOPSLA 2014): output i of the stream with state ``key`` is
  ``mix64(key + (i + 1) * 0x9E3779B97F4A7C15)`` with the published
  ``mix64`` finaliser.  Every draw is therefore addressable by
  (key, counter) and independent of how the work is chunked.
* Uniforms in [0, 1) take the top 53 bits.  Normals use the Box-Muller
  transform on consecutive uniform pairs (both the cosine and sine output).
* fp64 draws are rounded ONCE to bf16 with round-to-nearest-even (exact
  significand rounding via frexp/rint/ldexp), so the oracle (which widens the
  bf16 bits exactly) and the GPU see identical bytes.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

_GOLDEN = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)

MASK_TOKEN = -1          # response positions still masked carry this id
K_INFINITE = 2**31 - 1   # "radius K = infinity": never refresh on distance


def _mix64(z):
    """SplitMix64 finaliser on uint64 scalars or arrays (wrapping arithmetic)."""
    with np.errstate(over="ignore"):
        z = np.asarray(z, dtype=np.uint64)
        z = (z ^ (z >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
        return z ^ (z >> np.uint64(31))


def _fnv1a64(text: str) -> int:
    h = 0xCBF29CE484222325
    for byte in text.encode("utf-8"):
        h ^= byte
        h = (h * 0x100000001B3) & 0xFFFFFFFFFFFFFFFF
    return h


def stream_key(*parts) -> np.uint64:
    """Derive a 64-bit stream key from integers and strings (order matters)."""
    k = np.uint64(0x243F6A8885A308D3)
    with np.errstate(over="ignore"):
        for p in parts:
            v = _fnv1a64(p) if isinstance(p, str) else (int(p) & 0xFFFFFFFFFFFFFFFF)
            k = _mix64(k ^ (np.uint64(v) + _GOLDEN))
    return np.uint64(k)


def raw64(key, start: int, n: int) -> np.ndarray:
    """Outputs start .. start+n-1 of the SplitMix64 stream with state ``key``."""
    with np.errstate(over="ignore"):
        i = np.arange(start + 1, start + n + 1, dtype=np.uint64)
        return _mix64(np.uint64(key) + i * _GOLDEN)


def uniform(key, n: int, start: int = 0) -> np.ndarray:
    """n uniforms in [0, 1) (53-bit)."""
    return (raw64(key, start, n) >> np.uint64(11)).astype(np.float64) * (2.0 ** -53)


def normal(key, n: int) -> np.ndarray:
    """n standard normal deviates (Box-Muller over consecutive uniform pairs)."""
    m = (n + 1) // 2
    u = uniform(key, 2 * m)
    u1 = 1.0 - u[0::2]                      # (0, 1]
    u2 = u[1::2]
    r = np.sqrt(-2.0 * np.log(u1))
    t = 2.0 * math.pi * u2
    out = np.empty(2 * m, dtype=np.float64)
    out[0::2] = r * np.cos(t)
    out[1::2] = r * np.sin(t)
    return out[:n]


# ----------------------------------------------------------------------------
# rounding and widening
# ----------------------------------------------------------------------------

def to_bf16_bits(x) -> np.ndarray:
    """Round fp64 values once to bf16 (round-to-nearest-even); return uint16 bits."""
    x = np.asarray(x, dtype=np.float64)
    m, e = np.frexp(x)                       # x = m * 2**e, 0.5 <= |m| < 1
    normal_r = np.ldexp(np.rint(np.ldexp(m, 8)), e - 8)
    tiny = np.abs(x) < 2.0 ** -126            # bf16 subnormal range: spacing 2**-133
    sub_r = np.ldexp(np.rint(np.ldexp(x, 133)), -133)
    r = np.where(tiny, sub_r, normal_r)
    with np.errstate(over="ignore"):
        f32 = r.astype(np.float32)           # exact: r is on the bf16 grid
    return (f32.view(np.uint32) >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f64(bits) -> np.ndarray:
    """Exact widening of bf16 bit patterns to fp64."""
    b = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return b.view(np.float32).astype(np.float64)


def to_f32(x) -> np.ndarray:
    """Round fp64 values once to fp32 (IEEE round-to-nearest-even)."""
    return np.asarray(x, dtype=np.float64).astype(np.float32)


# ----------------------------------------------------------------------------
# workload recipes
# ----------------------------------------------------------------------------

@dataclass(frozen=True)
class AttnShape:
    batch: int
    prompt_len: int
    resp_len: int
    n_heads: int
    n_kv_heads: int
    head_dim: int

    @property
    def total_len(self) -> int:
        return self.prompt_len + self.resp_len


def bf16_normal(key_parts, shape, std: float) -> np.ndarray:
    """N(0, std^2) draws rounded once to bf16; returns uint16 bits of ``shape``."""
    n = int(np.prod(shape))
    return to_bf16_bits(normal(stream_key(*key_parts), n) * std).reshape(shape)


def attn_inputs(shape: AttnShape, seed: int = 0, std: float | None = None,
                layer: int = 0, step: int = 0) -> dict:
    """One layer's attention operands as bf16 bits.

    q_all  [B, N, Hq, D]   queries of all N = P + G positions (response queries
                           are rows P..N-1)
    k_prompt, v_prompt [B, P, Hkv, D]   prompt K/V under the current response
    k_cache,  v_cache  [B, P, Hkv, D]   prompt K/V under an older anchor response
    k_resp,   v_resp   [B, G, Hkv, D]   response K/V under the current response
    Values are N(0, 1) * std, std defaulting to 1/sqrt(D).
    """
    B, P, G = shape.batch, shape.prompt_len, shape.resp_len
    Hq, Hkv, D = shape.n_heads, shape.n_kv_heads, shape.head_dim
    N = P + G
    if std is None:
        std = 1.0 / math.sqrt(D)
    tag = ("attn", seed, layer, step)
    return {
        "q_all": bf16_normal(tag + ("q",), (B, N, Hq, D), std),
        "k_prompt": bf16_normal(tag + ("kp",), (B, P, Hkv, D), std),
        "v_prompt": bf16_normal(tag + ("vp",), (B, P, Hkv, D), std),
        "k_cache": bf16_normal(tag + ("kc",), (B, P, Hkv, D), std),
        "v_cache": bf16_normal(tag + ("vc",), (B, P, Hkv, D), std),
        "k_resp": bf16_normal(tag + ("kg",), (B, G, Hkv, D), std),
        "v_resp": bf16_normal(tag + ("vg",), (B, G, Hkv, D), std),
    }


def logits(rows: int, vocab: int, seed: int = 0, std: float = 2.5,
           boost_max: float = 0.0, dtype: str = "bf16", step: int = 0):
    """Vocabulary logits [rows, vocab]: N(0, std^2), plus (if boost_max > 0) one
    planted token per row, uniform over the vocabulary, boosted by U(0, boost_max).
    Returns uint16 bf16 bits or a float32 array."""
    z = normal(stream_key("logits", seed, step, rows, vocab), rows * vocab) * std
    z = z.reshape(rows, vocab)
    if boost_max > 0.0:
        u = uniform(stream_key("plant", seed, step, rows, vocab), 2 * rows)
        ids = np.minimum((u[0::2] * vocab).astype(np.int64), vocab - 1)
        z[np.arange(rows), ids] += u[1::2] * boost_max
    if dtype == "bf16":
        return to_bf16_bits(z)
    if dtype == "f32":
        return to_f32(z)
    raise ValueError(dtype)


def mask_state(batch: int, resp_len: int, seed: int = 0, frac: float = 0.5) -> np.ndarray:
    """uint8 [B, G]: 1 where the response position is still masked (Bernoulli(frac))."""
    u = uniform(stream_key("mask", seed, batch, resp_len), batch * resp_len)
    return (u < frac).astype(np.uint8).reshape(batch, resp_len)


def tokens(batch: int, resp_len: int, vocab: int, seed: int = 0,
           mask: np.ndarray | None = None) -> np.ndarray:
    """int32 [B, G] response token ids, uniform over the vocabulary; MASK_TOKEN
    where ``mask`` is set."""
    u = uniform(stream_key("tokens", seed, batch, resp_len, vocab), batch * resp_len)
    g = np.minimum((u * vocab).astype(np.int64), vocab - 1).astype(np.int32)
    g = g.reshape(batch, resp_len)
    if mask is not None:
        g = np.where(mask.astype(bool), np.int32(MASK_TOKEN), g).astype(np.int32)
    return g


def redraw_positions(seed: int, step: int, seq: int, resp_len: int, n: int) -> np.ndarray:
    """n distinct response positions, uniform without replacement, sorted."""
    u = raw64(stream_key("redraw-pos", seed, step, seq), 0, resp_len)
    return np.sort(np.argsort(u, kind="stable")[:n]).astype(np.int64)


def redraw_tokens(seed: int, step: int, seq: int, current: np.ndarray, vocab: int) -> np.ndarray:
    """A new id per position, uniform over the vocabulary minus the current id
    (uniform over the whole vocabulary where the current id is MASK_TOKEN)."""
    u = uniform(stream_key("redraw-tok", seed, step, seq), len(current))
    cur = np.asarray(current, dtype=np.int64)
    new = np.empty_like(cur)
    masked = cur < 0
    full = np.minimum((u * vocab).astype(np.int64), vocab - 1)
    less = np.minimum((u * (vocab - 1)).astype(np.int64), vocab - 2)
    new[masked] = full[masked]
    skip = ~masked
    new[skip] = np.where(less[skip] >= cur[skip], less[skip] + 1, less[skip])
    return new.astype(np.int32)


def redraw_rows(seed: int, step: int, layer: int, what: str, shape, std: float) -> np.ndarray:
    """Fresh bf16 rows for redrawn response positions (Q, K or V of one layer)."""
    return bf16_normal(("redraw-rows", seed, step, layer, what), shape, std)


@dataclass(frozen=True)
class Workload:
    """One named synthetic workload (shapes, distributions and schedule)."""
    name: str
    shape: AttnShape
    layers: int = 1
    steps: int = 1
    redraws_per_step: int = 0
    radius_k: int = K_INFINITE
    max_age: int = 0
    vocab: int = 0
    logits_rows: int = 0
    logits_dtype: str = "bf16"
    logits_std: float = 2.5
    logits_boost: float = 0.0
    notes: str = field(default="", compare=False)


WORKLOADS = {
    # batch 1, 1 layer, 4 = 4 heads, D 64, P 128, G 64; fp32 logits N(0, 9)
    # [64 x 1024]; 8 steps, 8 positions redrawn per step; refresh every 4 steps.
    "tiny": Workload("tiny", AttnShape(1, 128, 64, 4, 4, 64), layers=1, steps=8,
                     redraws_per_step=8, radius_k=K_INFINITE, max_age=4, vocab=1024,
                     logits_rows=64, logits_dtype="f32", logits_std=3.0),
    # LLaDA-8B-shaped layer: 32 = 32 heads, D 128, P 512, G 256; one step.
    "llada_layer": Workload("llada_layer", AttnShape(1, 512, 256, 32, 32, 128)),
    # decoder scoring: [4 x 256 x 126464] bf16 N(0, 2.5^2) + planted U(0, 6).
    "scoring": Workload("scoring", AttnShape(4, 0, 256, 1, 1, 128), vocab=126464,
                        logits_rows=4 * 256, logits_boost=6.0),
    # 32-layer trajectory: B 8, 32 heads, D 128, P 1024, G 512, 64 steps, 5%
    # redraw (26 of 512) per step, refresh at age 8 or distance > 64.
    "traj32": Workload("traj32", AttnShape(8, 1024, 512, 32, 32, 128), layers=32,
                       steps=64, redraws_per_step=26, radius_k=65, max_age=8,
                       vocab=126464),
    # long-prompt GQA: B 16, 28 q / 4 kv heads, D 128, P 4096, G 512, 32 layers
    # x 32 steps, 5% redraw, refresh every 16 steps, logits [16 x 512 x 152064].
    "gqa_long": Workload("gqa_long", AttnShape(16, 4096, 512, 28, 4, 128), layers=32,
                         steps=32, redraws_per_step=26, radius_k=K_INFINITE,
                         max_age=16, vocab=152064, logits_rows=16 * 512),
}


# ----------------------------------------------------------------------------
# device-side draws for full-size workloads (too large to draw on the host)
# ----------------------------------------------------------------------------

def device_normal(key_parts, shape, std: float, device, dtype=None):
    """N(0, std^2) draws made on the device by torch's seeded Philox generator
    (fp32, then rounded once to ``dtype``, bf16 by default).  Deterministic for
    a given key, shape and device type; used where the host generator would be
    too slow.  Callers that need oracle values copy the drawn tensor back."""
    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed(int(stream_key(*key_parts)) & 0x7FFFFFFFFFFFFFFF)
    x = torch.randn(tuple(shape), generator=gen, device=device, dtype=torch.float32)
    if std != 1.0:
        x.mul_(std)
    return x.to(torch.bfloat16 if dtype is None else dtype)


def device_attn_inputs(shape: AttnShape, device, seed: int = 0, std: float | None = None,
                       layer: int = 0, step: int = 0) -> dict:
    """attn_inputs' tensors drawn on the device (bf16 torch tensors)."""
    B, P, G = shape.batch, shape.prompt_len, shape.resp_len
    Hq, Hkv, D = shape.n_heads, shape.n_kv_heads, shape.head_dim
    if std is None:
        std = 1.0 / math.sqrt(D)
    tag = ("dev-attn", seed, layer, step)
    return {
        "q_all": device_normal(tag + ("q",), (B, P + G, Hq, D), std, device),
        "k_prompt": device_normal(tag + ("kp",), (B, P, Hkv, D), std, device),
        "v_prompt": device_normal(tag + ("vp",), (B, P, Hkv, D), std, device),
        "k_cache": device_normal(tag + ("kc",), (B, P, Hkv, D), std, device),
        "v_cache": device_normal(tag + ("vc",), (B, P, Hkv, D), std, device),
        "k_resp": device_normal(tag + ("kg",), (B, G, Hkv, D), std, device),
        "v_resp": device_normal(tag + ("vg",), (B, G, Hkv, D), std, device),
    }


def device_logits(rows: int, vocab: int, device, seed: int = 0, std: float = 2.5,
                  boost_max: float = 0.0, dtype=None, step: int = 0, row_stride: int | None = None):
    """logits' recipe drawn on the device: [rows, row_stride] (stride >= vocab;
    padding columns hold -inf and are never scored)."""
    import torch
    stride = vocab if row_stride is None else row_stride
    z = device_normal(("dev-logits", seed, step, rows, vocab), (rows, vocab), std, device, torch.float32)
    if boost_max > 0.0:
        gen = torch.Generator(device=device)
        gen.manual_seed(int(stream_key("dev-plant", seed, step, rows, vocab)) & 0x7FFFFFFFFFFFFFFF)
        ids = torch.randint(0, vocab, (rows,), generator=gen, device=device)
        boost = torch.rand(rows, generator=gen, device=device) * boost_max
        z[torch.arange(rows, device=device), ids] += boost
    out = torch.full((rows, stride), float("-inf"), device=device,
                     dtype=torch.bfloat16 if dtype is None else dtype)
    out[:, :vocab] = z.to(out.dtype)
    return out


# ----------------------------------------------------------------------------
# trajectory inputs (Algorithm 1 with the rollback decoder replaced by a
# seeded redraw).  Step 0 builds the cache; at step t >= 1, n positions per
# sequence get a new token id and new Q/K/V rows in every layer.  Fresh prompt
# Q/K/V (the stand-in for the model's prompt states under the current
# response) are drawn per (layer, step) and used only when a refresh fires.
# ----------------------------------------------------------------------------

def traj_initial_tokens(wl: Workload, seed: int = 0) -> np.ndarray:
    sh = wl.shape
    m = mask_state(sh.batch, sh.resp_len, seed=seed)
    return tokens(sh.batch, sh.resp_len, max(wl.vocab, 2), seed=seed, mask=m)


def traj_layer_initial(wl: Workload, seed: int, layer: int) -> dict:
    """Step-0 bits of one layer: q_all [B,N,Hq,D], k_resp/v_resp [B,G,Hkv,D],
    k_new/v_new [B,P,Hkv,D] (the fresh prompt K/V of the build)."""
    x = attn_inputs(wl.shape, seed=seed, layer=layer, step=0)
    return {"q_all": x["q_all"], "k_resp": x["k_resp"], "v_resp": x["v_resp"],
            "k_new": x["k_prompt"], "v_new": x["v_prompt"]}


def traj_redraw(wl: Workload, seed: int, step: int, g_current: np.ndarray):
    """Positions [B, n] (sorted, distinct) and their new token ids [B, n]."""
    B, G = g_current.shape
    n = wl.redraws_per_step
    pos = np.stack([redraw_positions(seed, step, b, G, n) for b in range(B)]) if n else np.zeros((B, 0), np.int64)
    new = np.stack([redraw_tokens(seed, step, b, g_current[b, pos[b]], max(wl.vocab, 2)) for b in range(B)]) \
        if n else np.zeros((B, 0), np.int32)
    return pos, new


def traj_redraw_rows(wl: Workload, seed: int, step: int, layer: int) -> dict:
    """New bf16 rows for the redrawn positions: q [B,n,Hq,D], k/v [B,n,Hkv,D]."""
    sh = wl.shape
    n = wl.redraws_per_step
    std = 1.0 / math.sqrt(sh.head_dim)
    return {"q": redraw_rows(seed, step, layer, "q", (sh.batch, n, sh.n_heads, sh.head_dim), std),
            "k": redraw_rows(seed, step, layer, "k", (sh.batch, n, sh.n_kv_heads, sh.head_dim), std),
            "v": redraw_rows(seed, step, layer, "v", (sh.batch, n, sh.n_kv_heads, sh.head_dim), std)}


def traj_fresh_prompt(wl: Workload, seed: int, step: int, layer: int) -> dict:
    """Fresh prompt queries [B,P,Hq,D] and K/V [B,P,Hkv,D] at a refresh of step t."""
    sh = wl.shape
    std = 1.0 / math.sqrt(sh.head_dim)
    tag = ("fresh-prompt", seed, step, layer)
    return {"q_prompt": bf16_normal(tag + ("q",), (sh.batch, sh.prompt_len, sh.n_heads, sh.head_dim), std),
            "k_new": bf16_normal(tag + ("k",), (sh.batch, sh.prompt_len, sh.n_kv_heads, sh.head_dim), std),
            "v_new": bf16_normal(tag + ("v",), (sh.batch, sh.prompt_len, sh.n_kv_heads, sh.head_dim), std)}


def traj_logits(wl: Workload, seed: int, step: int):
    """Logits scored after the forward of step t: [B*G, V] bf16 bits or fp32."""
    return logits(wl.shape.batch * wl.shape.resp_len, wl.vocab, seed=seed, std=wl.logits_std,
                  boost_max=wl.logits_boost, dtype=wl.logits_dtype, step=step)


# ----------------------------------------------------------------------------
# closed-loop decoding: the rollback decoder D is a confidence rule on the
# scores of the previous step's logits (oracle.decoder_update and
# archer_decoder_update); the logits plant a per-position target token whose
# boost grows with the step, so positions become confident at different steps
# and early guesses that are not the target get rolled back.
# ----------------------------------------------------------------------------

# decoder thresholds and the logits' boost growth used by closed-loop runs
CLOSED_LOOP = {"tau_accept": 0.9, "tau_remask": 0.05, "boost_per_step": 1.75}


def closed_loop_targets(wl: Workload, seed: int = 0):
    """Per-position target token [B, G] and boost rate [B, G] (U(0.5, 1.5))."""
    B, G = wl.shape.batch, wl.shape.resp_len
    u = uniform(stream_key("cl-target", seed, B, G), B * G)
    tgt = np.minimum((u * wl.vocab).astype(np.int64), wl.vocab - 1).astype(np.int32).reshape(B, G)
    rate = 0.5 + uniform(stream_key("cl-rate", seed, B, G), B * G).reshape(B, G)
    return tgt, rate


def closed_loop_logits(wl: Workload, seed: int, step: int, boost_per_step: float):
    """Logits scored after the forward of step t: N(0, std^2) plus
    boost_per_step * t * rate on each position's target token; bf16 bits or fp32."""
    B, G, V = wl.shape.batch, wl.shape.resp_len, wl.vocab
    z = normal(stream_key("cl-logits", seed, step, B, G, V), B * G * V).reshape(B * G, V) * wl.logits_std
    tgt, rate = closed_loop_targets(wl, seed)
    z[np.arange(B * G), tgt.reshape(-1)] += boost_per_step * step * rate.reshape(-1)
    if wl.logits_dtype == "bf16":
        return to_bf16_bits(z)
    return z.astype(np.float32)


def closed_loop_rows(wl: Workload, seed: int, step: int, layer: int) -> dict:
    """Candidate rows for every response position at step t (a changed position
    takes its own): q [B,G,Hq,D], k/v [B,G,Hkv,D] bf16 bits."""
    sh = wl.shape
    std = 1.0 / math.sqrt(sh.head_dim)
    B, G = sh.batch, sh.resp_len
    return {"q": bf16_normal(("cl-rows", seed, step, layer, "q"), (B, G, sh.n_heads, sh.head_dim), std),
            "k": bf16_normal(("cl-rows", seed, step, layer, "k"), (B, G, sh.n_kv_heads, sh.head_dim), std),
            "v": bf16_normal(("cl-rows", seed, step, layer, "v"), (B, G, sh.n_kv_heads, sh.head_dim), std)}


# ----------------------------------------------------------------------------
# staleness experiment: a synthetic prompt-cache map C_p(g) that is linear in
# the response embeddings E(g), so that Eq. theory-smoothness holds with a
# known constant:  K_p(g) = K_0 + alpha E(g) A_K^T,  V_p(g) = V_0 + alpha E(g) A_V^T
# (alpha [P, G], E(g) [G, d_e] one unit-norm embedding per token id, A [Hkv D, d_e]).
# ----------------------------------------------------------------------------

def staleness_model(shape: AttnShape, seed: int = 0, n_tokens: int = 64, d_e: int = 16,
                    drift: float = 0.6) -> dict:
    """Random pieces of the linear prompt-cache map (fp64) plus the layer's
    response queries and K/V (bf16 bits).  n_tokens embeddings (the last one is
    MASK_TOKEN's), rows normalised to 1; alpha ~ N(0, 1/G), A ~ N(0, 1/d_e),
    scaled by drift / sqrt(D) so that changing every position moves K_p by
    about drift times the spread of K_0."""
    B, P, G, Hq, Hkv, D = (shape.batch, shape.prompt_len, shape.resp_len, shape.n_heads, shape.n_kv_heads,
                           shape.head_dim)
    emb = normal(stream_key("st-emb", seed, n_tokens, d_e), n_tokens * d_e).reshape(n_tokens, d_e)
    emb /= np.linalg.norm(emb, axis=1, keepdims=True)
    alpha = normal(stream_key("st-alpha", seed, P, G), P * G).reshape(P, G) / math.sqrt(G)
    c = drift / math.sqrt(D)
    a_k = normal(stream_key("st-ak", seed, Hkv, D, d_e), Hkv * D * d_e).reshape(Hkv * D, d_e) * c / math.sqrt(d_e)
    a_v = normal(stream_key("st-av", seed, Hkv, D, d_e), Hkv * D * d_e).reshape(Hkv * D, d_e) * c / math.sqrt(d_e)
    x = attn_inputs(shape, seed=seed)
    return {"emb": emb, "alpha": alpha, "a_k": a_k, "a_v": a_v,
            "k0": bf16_bits_to_f64(x["k_cache"]), "v0": bf16_bits_to_f64(x["v_cache"]),
            "q_resp": x["q_all"][:, P:], "k_resp": x["k_resp"], "v_resp": x["v_resp"]}


def staleness_tokens(seed: int, batch: int, resp_len: int, n_tokens: int = 64) -> np.ndarray:
    """Anchor response g_r [B, G]: ids in [0, n_tokens - 1) (the last id is MASK's)."""
    u = uniform(stream_key("st-g", seed, batch, resp_len), batch * resp_len)
    return np.minimum((u * (n_tokens - 1)).astype(np.int64), n_tokens - 2).reshape(batch, resp_len)


def staleness_drift(g_r: np.ndarray, n_changed: int, seed: int, n_tokens: int = 64) -> np.ndarray:
    """g_t at Hamming distance n_changed from g_r in every sequence.  The drift
    is nested: a fixed seeded order of positions and a fixed new id per
    position (another id, uniform over the remaining ones); distance D changes
    the first D positions of that order."""
    B, G = g_r.shape
    g = g_r.copy()
    for b in range(B):
        u = raw64(stream_key("st-pos", seed, b), 0, G)
        pos = np.argsort(u, kind="stable")[:n_changed]
        v = uniform(stream_key("st-new", seed, b), G)[pos]
        shift = 1 + np.minimum((v * (n_tokens - 1)).astype(np.int64), n_tokens - 2)
        g[b, pos] = (g[b, pos] + shift) % n_tokens
    return g


def staleness_prompt_cache(model: dict, g: np.ndarray, Hkv: int, D: int):
    """K_p(g), V_p(g) [B, P, Hkv, D] in fp64 (the exact map; callers round to
    bf16 where the kernels need bf16)."""
    ae = np.einsum("pg,bge->bpe", model["alpha"], model["emb"][g])      # [B, P, d_e]
    dk = np.einsum("bpe,ce->bpc", ae, model["a_k"])
    dv = np.einsum("bpe,ce->bpc", ae, model["a_v"])
    B, P = g.shape[0], model["alpha"].shape[0]
    return (model["k0"] + dk.reshape(B, P, Hkv, D), model["v0"] + dv.reshape(B, P, Hkv, D))
