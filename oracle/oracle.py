"""ctypes binding of the fp64 Archer oracle (archer_oracle.cpp).

TEST INFRASTRUCTURE ONLY: imported by tests/, __graft_entry__.smoke() and the
CPU-baseline leg of bench.py, never by the CUDA path.  Inputs are numpy arrays
that the caller has widened exactly to float64 (bf16 bits -> fp64 with
``synth.bf16_bits_to_f64``); outputs are float64 / int32 numpy arrays.

What each function computes, and the passage it follows, is stated in the C++
source; the pins that fix it independently are in tests/test_oracle_pins.py.
"""
from __future__ import annotations

import ctypes
import hashlib
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "archer_oracle.cpp")
_BUILD = os.path.join(_HERE, "_build")
_lock = threading.Lock()
_lib = None

_dp = ctypes.POINTER(ctypes.c_double)
_ip = ctypes.POINTER(ctypes.c_int32)
_up = ctypes.POINTER(ctypes.c_uint8)


def build(force: bool = False) -> str:
    """Compile the oracle with g++ (portable C++17, no target-specific flags)."""
    with open(_SRC, "rb") as f:
        digest = hashlib.sha256(f.read()).hexdigest()[:16]
    os.makedirs(_BUILD, exist_ok=True)
    out = os.path.join(_BUILD, f"liboracle_{digest}.so")
    if force or not os.path.exists(out):
        tmp = out + f".tmp{os.getpid()}"
        subprocess.run(["g++", "-O2", "-std=c++17", "-fPIC", "-shared", "-pthread",
                        _SRC, "-o", tmp], check=True)
        os.replace(tmp, out)
    return out


def lib():
    global _lib
    with _lock:
        if _lib is None:
            L = ctypes.CDLL(build())
            L.oracle_attention.argtypes = [ctypes.c_int] * 7 + [ctypes.c_double] + [_dp] * 5 + [
                _ip, _dp, _dp, ctypes.c_int]
            L.oracle_attn_step.argtypes = [ctypes.c_int] * 6 + [ctypes.c_double] + [_dp] * 7 + [
                ctypes.c_int]
            L.oracle_prompt_refresh.argtypes = [ctypes.c_int] * 6 + [ctypes.c_double] + [_dp] * 9 + [
                _up, ctypes.c_int]
            L.oracle_attention_probs.argtypes = [ctypes.c_int] * 5 + [ctypes.c_double] + [_dp] * 5 + [
                ctypes.c_int, _dp]
            L.oracle_decode_scores.argtypes = [ctypes.c_int, ctypes.c_int, _dp, ctypes.c_int64, _up, _ip,
                                               _dp, _ip, _dp, _ip, _dp, ctypes.c_int]
            L.oracle_should_refresh.argtypes = [ctypes.c_int, ctypes.c_int, _ip, _ip, _ip, ctypes.c_int,
                                                ctypes.c_int, ctypes.c_int, _ip, _up]
            for name in ("oracle_attention", "oracle_attn_step", "oracle_prompt_refresh",
                         "oracle_attention_probs", "oracle_decode_scores", "oracle_should_refresh",
                         "oracle_hardware_threads"):
                getattr(L, name).restype = ctypes.c_int
            _lib = L
    return _lib


def _f64(a):
    return np.ascontiguousarray(a, dtype=np.float64)


def _ptr(a, t):
    return None if a is None else a.ctypes.data_as(t)


def _check(rc):
    if rc != 0:
        raise ValueError(f"oracle rejected its arguments (rc={rc})")


def hardware_threads() -> int:
    return int(lib().oracle_hardware_threads())


def attention(q, kp, vp, kg, vg, scale, row_begin=None, n_threads=0):
    """Attention of q [B, M, Hq, D] over [kp || kg], [vp || vg] (kp [B, P, Hkv, D],
    kg [B, G, Hkv, D]).  Returns (out [B, M, Hq, D], lse [B, Hq, M])."""
    q, kp, vp, kg, vg = map(_f64, (q, kp, vp, kg, vg))
    B, M, Hq, D = q.shape
    P, Hkv = kp.shape[1], kp.shape[2]
    G = kg.shape[1]
    out = np.zeros_like(q)
    lse = np.zeros((B, Hq, M))
    rb = None if row_begin is None else np.ascontiguousarray(row_begin, dtype=np.int32)
    _check(lib().oracle_attention(B, M, P, G, Hq, Hkv, D, float(scale), _ptr(q, _dp), _ptr(kp, _dp),
                                  _ptr(vp, _dp), _ptr(kg, _dp), _ptr(vg, _dp), _ptr(rb, _ip),
                                  _ptr(out, _dp), _ptr(lse, _dp), n_threads))
    return out, lse


def attn_step(q_resp, k_cache, v_cache, k_resp, v_resp, scale, n_threads=0):
    """Cached step: response queries over [cache || response].  Returns (out, lse)."""
    q, kc, vc, kg, vg = map(_f64, (q_resp, k_cache, v_cache, k_resp, v_resp))
    B, G, Hq, D = q.shape
    P, Hkv = kc.shape[1], kc.shape[2]
    out = np.zeros_like(q)
    lse = np.zeros((B, Hq, G))
    _check(lib().oracle_attn_step(B, P, G, Hq, Hkv, D, float(scale), _ptr(q, _dp), _ptr(kc, _dp),
                                  _ptr(vc, _dp), _ptr(kg, _dp), _ptr(vg, _dp), _ptr(out, _dp),
                                  _ptr(lse, _dp), n_threads))
    return out, lse


def prompt_refresh(q_all, k_new, v_new, k_resp, v_resp, k_cache, v_cache, scale, flags=None,
                   out=None, lse=None, n_threads=0):
    """Prompt refresh with optional per-sequence flags.  Returns
    (out [B, N, Hq, D], lse [B, Hq, N], k_cache', v_cache').  Rows a cleared flag
    leaves untouched keep the values of ``out`` / ``lse`` passed in (zeros by default)."""
    q, kn, vn, kg, vg = map(_f64, (q_all, k_new, v_new, k_resp, v_resp))
    kc = np.array(k_cache, dtype=np.float64, copy=True)
    vc = np.array(v_cache, dtype=np.float64, copy=True)
    B, N, Hq, D = q.shape
    P, Hkv = kn.shape[1], kn.shape[2]
    G = N - P
    o = np.zeros_like(q) if out is None else np.array(out, dtype=np.float64, copy=True)
    l = np.zeros((B, Hq, N)) if lse is None else np.array(lse, dtype=np.float64, copy=True)
    fl = None if flags is None else np.ascontiguousarray(flags, dtype=np.uint8)
    _check(lib().oracle_prompt_refresh(B, P, G, Hq, Hkv, D, float(scale), _ptr(q, _dp), _ptr(kn, _dp),
                                       _ptr(vn, _dp), _ptr(kg, _dp), _ptr(vg, _dp), _ptr(o, _dp),
                                       _ptr(l, _dp), _ptr(kc, _dp), _ptr(vc, _dp), _ptr(fl, _up),
                                       n_threads))
    return o, l, kc, vc


def attention_probs(q_row, kp, vp, kg, vg, h, n_heads, scale):
    """Explicit softmax row over [prompt || response] keys for one query row of
    head h (of n_heads); kp/vp are one sequence's [P, Hkv, D], kg/vg [G, Hkv, D]."""
    q_row, kp, vp, kg, vg = map(_f64, (q_row, kp, vp, kg, vg))
    P, Hkv, D = kp.shape
    G = kg.shape[0]
    probs = np.zeros(P + G)
    _check(lib().oracle_attention_probs(P, G, int(n_heads), Hkv, D, float(scale), _ptr(q_row, _dp),
                                        _ptr(kp, _dp), _ptr(vp, _dp), _ptr(kg, _dp), _ptr(vg, _dp),
                                        int(h), _ptr(probs, _dp)))
    return probs


def decode_scores(z, mask_state=None, cur_tokens=None, n_threads=0):
    """Scoring of logits z [rows, V] (any float dtype, widened exactly).
    Returns dict(max_prob, top1, margin, top2, cur_prob)."""
    z = _f64(z)
    rows, V = z.shape
    mp = np.zeros(rows)
    t1 = np.zeros(rows, dtype=np.int32)
    mg = np.zeros(rows)
    t2 = np.zeros(rows, dtype=np.int32)
    cp = np.zeros(rows)
    ms = None if mask_state is None else np.ascontiguousarray(mask_state, dtype=np.uint8).reshape(-1)
    ct = None if cur_tokens is None else np.ascontiguousarray(cur_tokens, dtype=np.int32).reshape(-1)
    _check(lib().oracle_decode_scores(rows, V, _ptr(z, _dp), V, _ptr(ms, _up), _ptr(ct, _ip),
                                      _ptr(mp, _dp), _ptr(t1, _ip), _ptr(mg, _dp), _ptr(t2, _ip),
                                      _ptr(cp, _dp), n_threads))
    return {"max_prob": mp, "top1": t1, "margin": mg, "top2": t2, "cur_prob": cp}


def should_refresh(g_cur, g_anchor, age, K, max_age, update_anchor=True):
    """Refresh rule.  Returns (dist, flag, g_anchor', age')."""
    g = np.ascontiguousarray(g_cur, dtype=np.int32)
    ga = np.array(g_anchor, dtype=np.int32, copy=True)
    ag = np.array(age, dtype=np.int32, copy=True)
    B, G = g.shape
    dist = np.zeros(B, dtype=np.int32)
    flag = np.zeros(B, dtype=np.uint8)
    _check(lib().oracle_should_refresh(B, G, _ptr(g, _ip), _ptr(ga, _ip), _ptr(ag, _ip), int(K),
                                       int(max_age), int(bool(update_anchor)), _ptr(dist, _ip),
                                       _ptr(flag, _up)))
    return dist, flag, ga, ag


def decoder_update(g, max_prob, top1, cur_prob, tau_accept, tau_remask, mask_token=-1):
    """Confidence-threshold rollback decoder, the synthetic stand-in for the
    decoder D of Algorithm 1 (Sec. 4.2; its decisions read the scoring
    outputs, the decoder-control inputs of Sec. 6).  Per sequence, from the
    scores of the previous step's logits:
      * a masked position whose max_prob >= tau_accept takes its top-1 token;
      * an unmasked position whose current token has probability
        cur_prob < tau_remask is masked again (rolled back);
      * if masked positions remain and none was accepted, the masked position
        with the largest max_prob (lowest index on ties) takes its top-1.
    Plain loops over positions; g [B, G] int32, scores [B * G].  Returns
    (g', changed [B, G] uint8)."""
    g = np.array(g, dtype=np.int32, copy=True)
    B, G = g.shape
    mp = np.asarray(max_prob, dtype=np.float64).reshape(B, G)
    t1 = np.asarray(top1, dtype=np.int64).reshape(B, G)
    cp = np.asarray(cur_prob, dtype=np.float64).reshape(B, G)
    changed = np.zeros((B, G), dtype=np.uint8)
    for b in range(B):
        accepted = False
        best, best_i = -1.0, -1
        old = g[b].copy()
        for i in range(G):
            if old[i] == mask_token:
                if mp[b, i] > best:
                    best, best_i = mp[b, i], i
                if mp[b, i] >= tau_accept:
                    g[b, i] = t1[b, i]
                    accepted = True
            elif cp[b, i] < tau_remask:
                g[b, i] = mask_token
        if not accepted and best_i >= 0:
            g[b, best_i] = t1[b, best_i]
        changed[b] = (g[b] != old).astype(np.uint8)
    return g, changed
