"""Pins of the fp64 oracle against what the paper and mathematics fix.

Each test checks the oracle against something other than itself: closed forms,
an independent high-precision (mpmath) evaluation written differently, exhaustive
enumeration, invariants, and the paper's own identities (refresh-every-step
equals eager decoding, Eq. archer-controller; dense rollback closure,
Prop. app-closure).  Every pin is chosen so that a plausible slip in the oracle
(dropped segment, wrong sign, wrong GQA index, transposed operand, scale applied
twice, wrong tie-break, off-by-one in the age rule) fails at least one test.
"""
import math

import mpmath
import numpy as np
import pytest

from oracle import oracle as O
from paper_2608_08086_gb300 import synth

mpmath.mp.dps = 40


def _rand_bf16(rng, shape, std=1.0):
    return synth.bf16_bits_to_f64(synth.to_bf16_bits(rng.standard_normal(shape) * std))


# ----------------------------------------------------------------------------
# attention (Sec. 4.1, Eq. archer-attention)
# ----------------------------------------------------------------------------

def _mp_attention(q, kp, vp, kg, vg, scale):
    """Independent evaluation with mpmath: p_j = exp(s_j) / sum_k exp(s_k) (no max
    shift), keys enumerated as prompt rows then response rows."""
    B, M, Hq, D = q.shape
    P, Hkv = kp.shape[1], kp.shape[2]
    G = kg.shape[1]
    grp = Hq // Hkv
    out = np.zeros((B, M, Hq, D))
    lse = np.zeros((B, Hq, M))
    for b in range(B):
        for h in range(Hq):
            kv = h // grp
            keys = [kp[b, j, kv] for j in range(P)] + [kg[b, j, kv] for j in range(G)]
            vals = [vp[b, j, kv] for j in range(P)] + [vg[b, j, kv] for j in range(G)]
            for i in range(M):
                ex = []
                for k in keys:
                    s = mpmath.mpf(0)
                    for c in range(D):
                        s += mpmath.mpf(float(q[b, i, h, c])) * mpmath.mpf(float(k[c]))
                    ex.append(mpmath.exp(mpmath.mpf(float(scale)) * s))
                tot = mpmath.fsum(ex)
                for c in range(D):
                    out[b, i, h, c] = float(mpmath.fsum(e * mpmath.mpf(float(v[c])) for e, v in zip(ex, vals)) / tot)
                lse[b, h, i] = float(mpmath.log(tot))
    return out, lse


@pytest.mark.parametrize("B,M,P,G,Hq,Hkv,D", [
    (1, 2, 3, 2, 2, 1, 3),
    (2, 3, 2, 3, 4, 2, 4),
    (1, 1, 0, 3, 2, 2, 2),      # P = 0: pure response self-attention
    (1, 4, 4, 1, 3, 1, 2),      # G = 1
])
def test_attention_matches_mpmath_brute_force(B, M, P, G, Hq, Hkv, D):
    rng = np.random.default_rng(1234 + B + M + P + G + Hq + D)
    q = _rand_bf16(rng, (B, M, Hq, D), 1.5)
    kp, vp = _rand_bf16(rng, (B, P, Hkv, D)), _rand_bf16(rng, (B, P, Hkv, D))
    kg, vg = _rand_bf16(rng, (B, G, Hkv, D)), _rand_bf16(rng, (B, G, Hkv, D))
    scale = 0.7
    out, lse = O.attention(q, kp, vp, kg, vg, scale)
    ref_out, ref_lse = _mp_attention(q, kp, vp, kg, vg, scale)
    np.testing.assert_allclose(out, ref_out, rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(lse, ref_lse, rtol=1e-12, atol=1e-13)


def test_attention_all_keys_equal_gives_mean_of_all_values():
    # Equal keys => uniform weights over BOTH segments => mean of all N values.
    rng = np.random.default_rng(0)
    B, P, G, Hq, Hkv, D = 2, 5, 3, 2, 2, 4
    k = rng.standard_normal(D)
    kp = np.broadcast_to(k, (B, P, Hkv, D)).copy()
    kg = np.broadcast_to(k, (B, G, Hkv, D)).copy()
    vp, vg = rng.standard_normal((B, P, Hkv, D)), rng.standard_normal((B, G, Hkv, D))
    q = rng.standard_normal((B, G, Hq, D))
    out, lse = O.attention(q, kp, vp, kg, vg, 0.3)
    mean = np.concatenate([vp, vg], axis=1).mean(axis=1)          # [B, Hkv, D]
    np.testing.assert_allclose(out, np.broadcast_to(mean[:, None], out.shape), rtol=1e-13, atol=1e-14)
    # lse = s + log N with s = scale * <q, k>
    s = 0.3 * np.einsum("bihd,d->bhi", q, k)
    np.testing.assert_allclose(lse, s + math.log(P + G), rtol=1e-13, atol=1e-13)


def test_attention_zero_query_is_uniform_mean():
    rng = np.random.default_rng(1)
    B, P, G, H, D = 1, 4, 4, 2, 3
    kp, vp = rng.standard_normal((B, P, H, D)), rng.standard_normal((B, P, H, D))
    kg, vg = rng.standard_normal((B, G, H, D)), rng.standard_normal((B, G, H, D))
    q = np.zeros((B, 2, H, D))
    out, lse = O.attention(q, kp, vp, kg, vg, 1.0)
    mean = np.concatenate([vp, vg], axis=1).mean(axis=1)
    np.testing.assert_allclose(out, np.broadcast_to(mean[:, None], out.shape), rtol=1e-13)
    np.testing.assert_allclose(lse, math.log(P + G), rtol=1e-14)


def test_attention_single_key_returns_its_value():
    rng = np.random.default_rng(2)
    q = rng.standard_normal((1, 3, 1, 4))
    kg, vg = rng.standard_normal((1, 1, 1, 4)), rng.standard_normal((1, 1, 1, 4))
    empty = np.zeros((1, 0, 1, 4))
    out, _ = O.attention(q, empty, empty, kg, vg, 1.0)
    np.testing.assert_allclose(out[0, :, 0], np.broadcast_to(vg[0, 0, 0], (3, 4)), rtol=1e-15)


def test_attention_two_keys_is_logistic():
    # Two keys: weight of key 1 = sigmoid(scale * <q, k1 - k2>) -- pins the scale and its sign.
    q = np.array([[[[1.0, -2.0]]]])
    kp = np.array([[[[0.5, 0.25]]]])       # prompt key
    kg = np.array([[[[-1.0, 0.75]]]])      # response key
    vp = np.array([[[[1.0, 0.0]]]])
    vg = np.array([[[[0.0, 1.0]]]])
    for scale in (0.125, 1.0, 3.0):
        out, lse = O.attention(q, kp, vp, kg, vg, scale)
        s1 = scale * (0.5 - 0.5)
        s2 = scale * (-1.0 - 1.5)
        w1 = 1.0 / (1.0 + math.exp(s2 - s1))
        assert abs(out[0, 0, 0, 0] - w1) < 1e-15
        assert abs(out[0, 0, 0, 1] - (1.0 - w1)) < 1e-15
        assert abs(lse[0, 0, 0] - (s1 + math.log1p(math.exp(s2 - s1)))) < 1e-14


def test_attention_dominant_key_selects_its_row():
    # One score far above the rest: out -> v_j* within exp(-gap) * (N - 1) * |v|.
    rng = np.random.default_rng(3)
    P, G, D = 6, 5, 4
    kp, vp = rng.standard_normal((1, P, 1, D)) * 0.1, rng.standard_normal((1, P, 1, D))
    kg, vg = rng.standard_normal((1, G, 1, D)) * 0.1, rng.standard_normal((1, G, 1, D))
    q = np.zeros((1, 1, 1, D))
    q[0, 0, 0, 0] = 1.0
    kg[0, 2, 0, 0] = 60.0                   # response row 2 dominates
    out, _ = O.attention(q, kp, vp, kg, vg, 1.0)
    np.testing.assert_allclose(out[0, 0, 0], vg[0, 2, 0], atol=1e-20 + 1e-22)
    kg[0, 2, 0, 0] = 0.0
    kp[0, 4, 0, 0] = 60.0                   # now prompt row 4 dominates
    out, _ = O.attention(q, kp, vp, kg, vg, 1.0)
    np.testing.assert_allclose(out[0, 0, 0], vp[0, 4, 0], atol=1e-20)


def test_attention_gqa_head_mapping():
    # Query head h reads KV head h // (Hq / Hkv): V constant per KV head tags it.
    B, P, G, Hq, Hkv, D = 1, 3, 2, 6, 3, 2
    rng = np.random.default_rng(4)
    kp, kg = rng.standard_normal((B, P, Hkv, D)), rng.standard_normal((B, G, Hkv, D))
    vp = np.zeros((B, P, Hkv, D))
    vg = np.zeros((B, G, Hkv, D))
    for kv in range(Hkv):
        vp[:, :, kv] = 10.0 * (kv + 1)
        vg[:, :, kv] = 10.0 * (kv + 1)
    q = rng.standard_normal((B, G, Hq, D))
    out, _ = O.attention(q, kp, vp, kg, vg, 1.0)
    for h in range(Hq):
        np.testing.assert_allclose(out[0, :, h], 10.0 * (h // 2 + 1), rtol=1e-14)


def test_attention_probability_rows_sum_to_one():
    sh = synth.AttnShape(1, 48, 32, 4, 2, 16)
    x = {k: synth.bf16_bits_to_f64(v) for k, v in synth.attn_inputs(sh, seed=7, std=1.0).items()}
    for h in range(4):
        for i in (0, 17, 79):
            p = O.attention_probs(x["q_all"][0, i, h], x["k_cache"][0], x["v_cache"][0],
                                  x["k_resp"][0], x["v_resp"][0], h, 4, 1.0 / 4.0)
            assert p.shape == (80,)
            assert np.all(p > 0)
            assert abs(p.sum() - 1.0) <= 1e-12


def test_attention_prob_row_matches_output():
    # out = sum_j p_j v_j with the explicit probability row (no transposed operand).
    sh = synth.AttnShape(1, 8, 8, 2, 1, 8)
    x = {k: synth.bf16_bits_to_f64(v) for k, v in synth.attn_inputs(sh, seed=8, std=1.0).items()}
    out, _ = O.attention(x["q_all"], x["k_prompt"], x["v_prompt"], x["k_resp"], x["v_resp"], 0.5)
    vcat = np.concatenate([x["v_prompt"][0, :, 0], x["v_resp"][0, :, 0]], axis=0)
    for h in range(2):
        for i in range(16):
            p = O.attention_probs(x["q_all"][0, i, h], x["k_prompt"][0], x["v_prompt"][0],
                                  x["k_resp"][0], x["v_resp"][0], h, 2, 0.5)
            np.testing.assert_allclose(out[0, i, h], p @ vcat, rtol=1e-13, atol=1e-15)


def test_refresh_every_step_equals_eager():
    # Eq. archer-controller: with the cache built from the current response
    # (D_t >= K branch), the cached forward IS the full forward on the response
    # rows.  The oracle must match bit for bit.
    sh = synth.AttnShape(2, 40, 24, 4, 2, 8)
    x = {k: synth.bf16_bits_to_f64(v) for k, v in synth.attn_inputs(sh, seed=11).items()}
    P = sh.prompt_len
    scale = 1.0 / math.sqrt(8)
    full, lse_f, kc, vc = O.prompt_refresh(x["q_all"], x["k_prompt"], x["v_prompt"], x["k_resp"],
                                           x["v_resp"], x["k_cache"], x["v_cache"], scale)
    np.testing.assert_array_equal(kc, x["k_prompt"])        # cache replaced by fresh K/V
    np.testing.assert_array_equal(vc, x["v_prompt"])
    step, lse_s = O.attn_step(x["q_all"][:, P:], kc, vc, x["k_resp"], x["v_resp"], scale)
    np.testing.assert_array_equal(step, full[:, P:])
    np.testing.assert_array_equal(lse_s, lse_f[:, :, P:])


def test_cached_step_reads_the_anchor_cache_not_the_fresh_prompt():
    # Eq. archer-cached: the step uses C_p(g_r); changing the fresh prompt K/V
    # must not change it, changing the cache must.
    sh = synth.AttnShape(1, 16, 8, 2, 2, 8)
    x = {k: synth.bf16_bits_to_f64(v) for k, v in synth.attn_inputs(sh, seed=12).items()}
    P = sh.prompt_len
    a, _ = O.attn_step(x["q_all"][:, P:], x["k_cache"], x["v_cache"], x["k_resp"], x["v_resp"], 0.35)
    ref, _ = _mp_attention(x["q_all"][:, P:P + 2], x["k_cache"], x["v_cache"], x["k_resp"], x["v_resp"], 0.35)
    np.testing.assert_allclose(a[:, :2], ref, rtol=1e-12, atol=1e-13)
    b, _ = O.attn_step(x["q_all"][:, P:], x["k_prompt"], x["v_prompt"], x["k_resp"], x["v_resp"], 0.35)
    assert np.abs(a - b).max() > 1e-3


def test_mixed_batch_refresh_flags():
    # Flagged sequences: N queries over the fresh prompt, cache replaced.
    # Unflagged: response rows over the old cache, prompt rows untouched, cache kept.
    sh = synth.AttnShape(3, 12, 8, 2, 1, 4)
    x = {k: synth.bf16_bits_to_f64(v) for k, v in synth.attn_inputs(sh, seed=13).items()}
    P, scale = sh.prompt_len, 0.5
    flags = np.array([1, 0, 1], dtype=np.uint8)
    sentinel = np.full(x["q_all"].shape, 7.0)
    out, lse, kc, vc = O.prompt_refresh(x["q_all"], x["k_prompt"], x["v_prompt"], x["k_resp"], x["v_resp"],
                                        x["k_cache"], x["v_cache"], scale, flags=flags, out=sentinel)
    full, _, _, _ = O.prompt_refresh(x["q_all"], x["k_prompt"], x["v_prompt"], x["k_resp"], x["v_resp"],
                                     x["k_cache"], x["v_cache"], scale)
    step, _ = O.attn_step(x["q_all"][:, P:], x["k_cache"], x["v_cache"], x["k_resp"], x["v_resp"], scale)
    for b in (0, 2):
        np.testing.assert_array_equal(out[b], full[b])
        np.testing.assert_array_equal(kc[b], x["k_prompt"][b])
    np.testing.assert_array_equal(out[1, P:], step[1])
    assert np.all(out[1, :P] == 7.0)
    np.testing.assert_array_equal(kc[1], x["k_cache"][1])
    np.testing.assert_array_equal(vc[1], x["v_cache"][1])


def test_dense_rollback_closure():
    # Prop. app-closure: changing one response position's K/V changes EVERY
    # query's output, prompt queries included (refresh mode).
    sh = synth.AttnShape(1, 10, 6, 2, 2, 4)
    x = {k: synth.bf16_bits_to_f64(v) for k, v in synth.attn_inputs(sh, seed=14, std=1.0).items()}
    args = (x["q_all"], x["k_prompt"], x["v_prompt"])
    base, _, _, _ = O.prompt_refresh(*args, x["k_resp"], x["v_resp"], x["k_cache"], x["v_cache"], 0.5)
    kg = x["k_resp"].copy()
    kg[0, 3] += 0.25
    pert, _, _, _ = O.prompt_refresh(*args, kg, x["v_resp"], x["k_cache"], x["v_cache"], 0.5)
    diff = np.abs(pert - base).max(axis=-1)            # [B, N, Hq]
    assert np.all(diff > 0), "a query row did not depend on the changed response key"
    vg = x["v_resp"].copy()
    vg[0, 5] += 0.25
    pert, _, _, _ = O.prompt_refresh(*args, x["k_resp"], vg, x["k_cache"], x["v_cache"], 0.5)
    assert np.all(np.abs(pert - base).max(axis=-1) > 0)


# ----------------------------------------------------------------------------
# decoder scoring
# ----------------------------------------------------------------------------

def _brute_scores(z):
    """Full stable sort of (-z, index) and mpmath softmax."""
    rows = []
    for r in z:
        order = sorted(range(len(r)), key=lambda j: (-r[j], j))
        ex = [mpmath.exp(mpmath.mpf(float(v))) for v in r]
        tot = mpmath.fsum(ex)
        p = [e / tot for e in ex]
        t1 = order[0]
        t2 = order[1] if len(r) > 1 else None
        rows.append((t1, float(p[t1]), float(p[t1] - (p[t2] if t2 is not None else 0)), t2,
                     float(mpmath.fsum(p))))
    return rows


def test_scores_match_sorted_brute_force_with_ties():
    rng = np.random.default_rng(5)
    z = rng.integers(-3, 4, size=(40, 9)).astype(np.float64) * 0.5   # many ties
    z[:, ::3] += rng.standard_normal((40, 3))
    res = O.decode_scores(z)
    for r, (t1, mp, mg, t2, tot) in enumerate(_brute_scores(z)):
        assert res["top1"][r] == t1
        assert res["top2"][r] == t2
        assert abs(res["max_prob"][r] - mp) < 1e-14
        assert abs(res["margin"][r] - mg) < 1e-14
        assert abs(tot - 1.0) < 1e-30


def test_scores_constant_row():
    V = 37
    res = O.decode_scores(np.full((2, V), 1.25))
    assert list(res["top1"]) == [0, 0]
    np.testing.assert_allclose(res["max_prob"], 1.0 / V, rtol=1e-14)
    np.testing.assert_array_equal(res["margin"], 0.0)


def test_scores_two_entries_logistic():
    for a, b in ((0.0, 1.0), (3.5, -2.0), (-1.0, -1.0)):
        res = O.decode_scores(np.array([[a, b]]))
        d = abs(a - b)
        assert res["top1"][0] == (1 if b > a else 0)
        assert abs(res["max_prob"][0] - 1.0 / (1.0 + math.exp(-d))) < 1e-15
        assert abs(res["margin"][0] - math.tanh(d / 2.0)) < 1e-15


def test_scores_planted_boost_dominates_and_minus_inf_is_zero():
    V = 1000
    z = np.zeros((1, V))
    z[0, 321] = 80.0
    res = O.decode_scores(z)
    assert res["top1"][0] == 321
    assert abs(res["max_prob"][0] - 1.0) < 1e-30 + (V - 1) * math.exp(-80.0) * 2
    z = np.full((1, 5), -np.inf)
    z[0, 2] = 0.0
    z[0, 4] = math.log(3.0)
    res = O.decode_scores(z)
    assert res["top1"][0] == 4 and res["top2"][0] == 2
    assert abs(res["max_prob"][0] - 0.75) < 1e-15
    assert abs(res["margin"][0] - 0.5) < 1e-15


def test_scores_single_entry_and_cur_prob_gating():
    res = O.decode_scores(np.array([[4.0]]))
    assert res["top1"][0] == 0 and res["max_prob"][0] == 1.0 and res["margin"][0] == 1.0
    z = np.log(np.array([[1.0, 2.0, 5.0], [1.0, 1.0, 2.0], [1.0, 1.0, 1.0]]))
    res = O.decode_scores(z, mask_state=np.array([0, 1, 0], np.uint8),
                          cur_tokens=np.array([1, 2, -1], np.int32))
    np.testing.assert_allclose(res["cur_prob"], [0.25, 0.0, 0.0], rtol=1e-15)


# ----------------------------------------------------------------------------
# refresh rule (Sec. 4.2, Eq. archer-distance / archer-controller; age signal of Sec. 6)
# ----------------------------------------------------------------------------

def test_refresh_rule_exhaustive_small():
    G = 4
    syms = np.array([-1, 0, 1], dtype=np.int32)            # MASK and two tokens
    grid = np.array(np.meshgrid(*([syms] * G), indexing="ij")).reshape(G, -1).T
    n = len(grid)
    g = np.repeat(grid, n, axis=0)
    ga = np.tile(grid, (n, 1))
    # brute-force distance: count the positions of the set {i : g_i != ga_i}
    brute_d = np.array([len({i for i in range(G) if gi[i] != ai[i]}) for gi, ai in zip(g, ga)])
    for K in (0, 1, 2, 3, 4, 5, synth.K_INFINITE):
        for max_age in (0, 1, 2, 4):
            for age0 in (0, 1, 3):
                age = np.full(len(g), age0, dtype=np.int32)
                d, f, ga2, age2 = O.should_refresh(g, ga, age, K, max_age, update_anchor=True)
                assert np.array_equal(d, brute_d)
                expect = (brute_d >= K) | ((max_age > 0) & (age0 + 1 >= max_age))
                assert np.array_equal(f.astype(bool), expect)
                assert np.array_equal(ga2[expect], g[expect])
                assert np.array_equal(ga2[~expect], ga[~expect])
                assert np.all(age2[expect] == 0) and np.all(age2[~expect] == age0 + 1)
                d3, f3, ga3, age3 = O.should_refresh(g, ga, age, K, max_age, update_anchor=False)
                assert np.array_equal(d3, brute_d) and np.array_equal(f3, f)
                assert np.array_equal(ga3, ga) and np.array_equal(age3, age)


def test_refresh_rule_paper_special_cases():
    rng = np.random.default_rng(6)
    g = rng.integers(0, 50, size=(64, 32)).astype(np.int32)
    ga = g.copy()
    flip = rng.random((64, 32)) < 0.1
    ga[flip] = (ga[flip] + 1) % 50
    age = np.zeros(64, np.int32)
    d, f, _, _ = O.should_refresh(g, ga, age, 1, 0)     # K = 1: any change refreshes
    assert np.array_equal(f.astype(bool), flip.any(axis=1))
    d, f, _, _ = O.should_refresh(g, ga, age, synth.K_INFINITE, 0)   # K = inf: never
    assert not f.any()
    d, f, _, _ = O.should_refresh(g, ga, age, 0, 0)     # K = 0: always
    assert f.all()
    # invariants of the Hamming distance: symmetry, identity, bound, triangle
    d_ab, _, _, _ = O.should_refresh(g, ga, age, 1, 0, False)
    d_ba, _, _, _ = O.should_refresh(ga, g, age, 1, 0, False)
    assert np.array_equal(d_ab, d_ba) and np.all(d_ab <= 32)
    d_aa, _, _, _ = O.should_refresh(g, g, age, 1, 0, False)
    assert not d_aa.any()
    gc = rng.integers(0, 50, size=(64, 32)).astype(np.int32)
    d_ac, _, _, _ = O.should_refresh(g, gc, age, 1, 0, False)
    d_cb, _, _, _ = O.should_refresh(gc, ga, age, 1, 0, False)
    assert np.all(d_ab <= d_ac + d_cb)


def test_age_schedule_refreshes_every_max_age_steps():
    # "every 4 steps": with no distance trigger, refresh at t = 4, 8 (age counted
    # from the build at t = 0).
    g = np.zeros((1, 8), np.int32)
    ga, age = g.copy(), np.zeros(1, np.int32)
    fired = []
    for t in range(1, 13):
        _, f, ga, age = O.should_refresh(g, ga, age, synth.K_INFINITE, 4)
        if f[0]:
            fired.append(t)
    assert fired == [4, 8, 12]


def test_net_distance_not_cumulative():
    # Eq. archer-distance counts net drift: a position that reverts counts 0.
    ga = np.array([[1, 2, 3, 4]], np.int32)
    _, _, _, _ = O.should_refresh(ga, ga, np.zeros(1, np.int32), 2, 0)
    g1 = np.array([[9, 2, 3, 4]], np.int32)
    d1, f1, ga1, age1 = O.should_refresh(g1, ga, np.zeros(1, np.int32), 2, 0)
    assert d1[0] == 1 and f1[0] == 0
    g2 = np.array([[1, 2, 3, 4]], np.int32)              # reverted
    d2, f2, _, _ = O.should_refresh(g2, ga1, age1, 2, 0)
    assert d2[0] == 0 and f2[0] == 0
