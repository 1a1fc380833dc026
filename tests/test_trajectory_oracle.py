"""Algorithm 1 on the oracle: schedules and identities the paper fixes.

* K = 1 with a change every step refreshes every step, so Archer's logits
  equal eager decoding's (Sec. 6 radius sweep: "at K = 1 ... approaches eager").
* K = infinity and no age cap: only the build refresh (the initial snapshot is
  never synchronised again).
* an age cap of 4 refreshes at t = 4, 8 ("every 4 steps").
* the 32-layer trajectory's rule (26 of 512 positions redrawn per step,
  refresh at age 8 or distance > 64) refreshes every third step: the expected
  number of distinct positions after two steps is 512 (1 - (1 - 26/512)^2) = 50.7
  < 65 and after three 74.0 >= 65, so q_K = 1/3 (the speedup model of
  Eq. app-speedup-exact then predicts 1 / (1/3 + 2/3 * G/N)).
"""
import dataclasses

import numpy as np

from oracle import oracle as O
from oracle import trajectory as OT
from paper_2608_08086_gb300 import synth

TINY = synth.WORKLOADS["tiny"]


def _refresh_steps(records):
    return [r["t"] for r in records if r["t"] > 0 and r["flag"].any()]


def test_tiny_workload_refreshes_every_four_steps():
    recs = OT.run(TINY, seed=0, score=False)
    assert _refresh_steps(recs) == [4, 8]
    assert len(recs) == TINY.steps + 1


def test_k1_equals_eager_bit_for_bit():
    wl = dataclasses.replace(TINY, radius_k=1, max_age=0, steps=4)
    archer = OT.run(wl, seed=1, score=False)
    eager = OT.run(wl, seed=1, mode="eager", score=False)
    assert _refresh_steps(archer) == [1, 2, 3, 4]
    for a, e in zip(archer, eager):
        for oa, oe in zip(a["out"], e["out"]):
            np.testing.assert_array_equal(oa, oe)


def test_k_infinite_never_refreshes_after_the_build():
    wl = dataclasses.replace(TINY, radius_k=synth.K_INFINITE, max_age=0, steps=6)
    recs = OT.run(wl, seed=2, score=False)
    assert _refresh_steps(recs) == []
    # cached steps read the build-time cache: the output differs from eager once
    # the response has drifted (the approximation Archer trades for speed)
    eager = OT.run(wl, seed=2, mode="eager", score=False)
    assert np.abs(recs[-1]["out"][0] - eager[-1]["out"][0][:, wl.shape.prompt_len:]).max() > 0


def test_cached_step_equals_eager_when_nothing_changed():
    # No redraw: g_t = g_r, so the cached forward IS the fresh forward.
    wl = dataclasses.replace(TINY, redraws_per_step=0, radius_k=synth.K_INFINITE, max_age=0, steps=2)
    recs = OT.run(wl, seed=3, score=False)
    P = wl.shape.prompt_len
    for r in recs[1:]:
        np.testing.assert_array_equal(r["out"][0], recs[0]["out"][0][:, P:])


def test_traj32_rule_refreshes_every_third_step():
    wl = synth.WORKLOADS["traj32"]
    B, G = wl.shape.batch, wl.shape.resp_len
    g = synth.traj_initial_tokens(wl, seed=0)
    ga, age = g.copy(), np.zeros(B, np.int32)
    fired = []
    dists = []
    for t in range(1, wl.steps + 1):
        pos, new = synth.traj_redraw(wl, 0, t, g)
        g[np.arange(B)[:, None], pos] = new
        d, f, ga, age = O.should_refresh(g, ga, age, wl.radius_k, wl.max_age)
        assert f.all() or not f.any()          # the batch stays in lock-step here
        dists.append(d)
        if f.all():
            fired.append(t)
    assert fired == list(range(3, wl.steps + 1, 3))
    q_k = (len(fired) + 1) / (wl.steps + 1)        # the build counts as a refresh
    assert abs(q_k - 1 / 3) < 0.02
    # distances just before a refresh are all >= 65, one step earlier all <= 52
    d = np.array(dists)
    assert d[2::3].min() >= 65 and d[1::3].max() <= 52


# A small batch whose sequences refresh at different steps, by distance and by
# the age cap (B 3, 2 q / 1 kv heads, D 16, P 16, G 24, 2 layers, 10 steps,
# 2 positions redrawn per step, K = 6, max_age = 4; with seed 2 six steps
# refresh part of the batch and the age cap alone fires twice).
MIXED = synth.Workload("mixed", synth.AttnShape(3, 16, 24, 2, 1, 16), layers=2, steps=10,
                       redraws_per_step=2, radius_k=6, max_age=4, vocab=50)


def test_trajectory_follows_the_definition_step_by_step():
    """Algorithm 1 restated per sequence from the definitions, without the
    driver's carried state, and compared with every record of the driver:
      * g_t: the redraws applied in step order;
      * the sequence's anchor step r (0 at the build) and D_t = Hamming(g_t, g_r)
        (Eq. archer-distance); refresh iff D_t >= K or t - r >= max_age;
      * a response row at step t is the row of the latest redraw of that
        position up to t (else the build's row), looked up, not carried;
      * the prompt cache a cached step reads is the fresh prompt K/V of step r
        (Eq. archer-cached); a refresh reads the fresh prompt of step t, and its
        prompt queries are that step's;
      * each output row is the oracle's attention over those inputs."""
    wl, seed = MIXED, 2
    sh = wl.shape
    B, P, G, D = sh.batch, sh.prompt_len, sh.resp_len, sh.head_dim
    scale = 1.0 / np.sqrt(D)
    f64 = synth.bf16_bits_to_f64
    recs = OT.run(wl, seed=seed, score=False)
    assert len(recs) == wl.steps + 1

    g = synth.traj_initial_tokens(wl, seed)
    states = [g.copy()]
    redraws = [None]                                   # step -> (pos [B, n], rows per layer)
    anchor = np.zeros(B, dtype=np.int64)               # anchor step r per sequence
    init = [synth.traj_layer_initial(wl, seed, layer) for layer in range(wl.layers)]
    fresh = {}

    def prompt_of(step, layer):
        if step == 0:
            return f64(init[layer]["k_new"]), f64(init[layer]["v_new"]), f64(init[layer]["q_all"][:, :P])
        if (step, layer) not in fresh:
            fp = synth.traj_fresh_prompt(wl, seed, step, layer)
            fresh[(step, layer)] = (f64(fp["k_new"]), f64(fp["v_new"]), f64(fp["q_prompt"]))
        return fresh[(step, layer)]

    def response_rows(t, layer, b):
        q = f64(init[layer]["q_all"][b, P:]).copy()
        k = f64(init[layer]["k_resp"][b]).copy()
        v = f64(init[layer]["v_resp"][b]).copy()
        for i in range(G):
            for s in range(t, 0, -1):                  # latest redraw of position i
                hit = np.nonzero(redraws[s][0][b] == i)[0]
                if hit.size:
                    rows = redraws[s][1][layer]
                    q[i], k[i], v[i] = f64(rows["q"][b, hit[0]]), f64(rows["k"][b, hit[0]]), f64(rows["v"][b, hit[0]])
                    break
        return q, k, v

    mixed_steps = cap_fires = 0
    for t in range(0, wl.steps + 1):
        rec = recs[t]
        if t == 0:
            flag = np.ones(B, dtype=bool)
        else:
            pos, new = synth.traj_redraw(wl, seed, t, g)
            g[np.arange(B)[:, None], pos] = new
            states.append(g.copy())
            redraws.append((pos, [synth.traj_redraw_rows(wl, seed, t, layer) for layer in range(wl.layers)]))
            dist = np.array([(g[b] != states[anchor[b]][b]).sum() for b in range(B)])
            flag = (dist >= wl.radius_k) | ((t - anchor) >= wl.max_age)
            np.testing.assert_array_equal(rec["dist"], dist)
            np.testing.assert_array_equal(rec["flag"].astype(bool), flag)
            mixed_steps += int(0 < flag.sum() < B)
            cap_fires += int((flag & (dist < wl.radius_k)).sum())
        any_refresh = bool(flag.any())
        for layer in range(wl.layers):
            out = rec["out"][layer]
            assert out.shape[1] == (P + G if any_refresh else G)
            for b in range(B):
                q, k, v = response_rows(t, layer, b)
                if flag[b]:
                    kp, vp, qp = prompt_of(t, layer)
                    qa = np.concatenate([qp[b], q])[None]
                    want, _ = O.attention(qa, kp[b][None], vp[b][None], k[None], v[None], scale)
                    np.testing.assert_allclose(out[b], want[0], rtol=1e-12, atol=1e-15)
                else:
                    kp, vp, _ = prompt_of(int(anchor[b]), layer)
                    want, _ = O.attention(q[None], kp[b][None], vp[b][None], k[None], v[None], scale)
                    got = out[b, P:] if any_refresh else out[b]
                    np.testing.assert_allclose(got, want[0], rtol=1e-12, atol=1e-15)
        anchor[flag] = t
    # the case exercises what it is meant to
    assert mixed_steps >= 3 and cap_fires >= 1
