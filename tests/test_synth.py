"""The seeded input generator: published SplitMix64 outputs, exact bf16 rounding,
determinism and the workload recipes' statistics."""
import numpy as np
import torch

from paper_2608_08086_gb300 import synth


def test_splitmix64_published_outputs():
    # SplitMix64 with state 0: the first three outputs of the reference generator.
    assert [int(x) for x in synth.raw64(0, 0, 3)] == [
        0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_stream_is_counter_addressable():
    k = synth.stream_key("x", 3)
    a = synth.raw64(k, 0, 100)
    b = synth.raw64(k, 40, 60)
    np.testing.assert_array_equal(a[40:], b)


def test_bf16_rounding_matches_torch_for_fp32_inputs():
    rng = np.random.default_rng(0)
    x = (rng.standard_normal(200_000) * 3.0).astype(np.float32).astype(np.float64)
    x = np.concatenate([x, [0.0, -0.0, 1.0, 1.00390625, 1.01171875, 2.0 ** -130, -3.0e38]])
    ours = synth.to_bf16_bits(x)
    theirs = torch.from_numpy(x.astype(np.float32)).to(torch.bfloat16).view(torch.int16).numpy()
    np.testing.assert_array_equal(ours, theirs.view(np.uint16))


def test_bf16_round_trip_and_ties_to_even():
    # 1 + 2^-8 lies halfway between 1 and 1 + 2^-7: ties go to the even significand (1.0).
    bits = synth.to_bf16_bits(np.array([1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8]))
    np.testing.assert_array_equal(synth.bf16_bits_to_f64(bits), [1.0, 1.0 + 2.0 ** -6])
    x = synth.bf16_bits_to_f64(synth.to_bf16_bits(np.linspace(-4, 4, 1001)))
    np.testing.assert_array_equal(synth.bf16_bits_to_f64(synth.to_bf16_bits(x)), x)


def test_normal_statistics():
    z = synth.normal(synth.stream_key("stats"), 400_000)
    assert abs(z.mean()) < 0.01
    assert abs(z.std() - 1.0) < 0.01


def test_redraw_positions_distinct_and_tokens_change():
    for step in range(5):
        pos = synth.redraw_positions(0, step, 3, 512, 26)
        assert len(set(pos.tolist())) == 26 and pos.min() >= 0 and pos.max() < 512
    cur = np.array([-1, 0, 5, 9, 9], dtype=np.int32)
    for step in range(50):
        new = synth.redraw_tokens(1, step, 0, cur, 10)
        assert np.all(new != cur) and np.all((new >= 0) & (new < 10))


def test_attn_inputs_deterministic_and_scaled():
    sh = synth.AttnShape(1, 64, 32, 2, 1, 64)
    a = synth.attn_inputs(sh, seed=5)
    b = synth.attn_inputs(sh, seed=5)
    for k in a:
        np.testing.assert_array_equal(a[k], b[k])
    q = synth.bf16_bits_to_f64(a["q_all"])
    assert abs(q.std() - 1.0 / 8.0) < 0.01
    assert a["q_all"].shape == (1, 96, 2, 64) and a["k_resp"].shape == (1, 32, 1, 64)


def test_logits_planted_token():
    z = synth.bf16_bits_to_f64(synth.logits(16, 4096, seed=1, std=2.5, boost_max=6.0))
    assert z.shape == (16, 4096)
    assert abs(z.std() - 2.5) < 0.1


def test_workloads_match_the_stated_recipe():
    # the shapes and schedules of the synthetic workloads (the paper's
    # code-generation settings: LLaDA-shaped layers, 5 % redraw per step,
    # refresh by distance K = 65 or by an age cap)
    W = synth.WORKLOADS
    want = {
        "tiny": ((1, 128, 64, 4, 4, 64), 1, 8, 8, synth.K_INFINITE, 4, 1024, 64, "f32"),
        "llada_layer": ((1, 512, 256, 32, 32, 128), 1, 1, 0, synth.K_INFINITE, 0, 0, 0, "bf16"),
        "scoring": ((4, 0, 256, 1, 1, 128), 1, 1, 0, synth.K_INFINITE, 0, 126464, 1024, "bf16"),
        "traj32": ((8, 1024, 512, 32, 32, 128), 32, 64, 26, 65, 8, 126464, 0, "bf16"),
        "gqa_long": ((16, 4096, 512, 28, 4, 128), 32, 32, 26, synth.K_INFINITE, 16, 152064, 16 * 512, "bf16"),
    }
    assert set(W) == set(want)
    for name, (shape, layers, steps, redraws, K, max_age, vocab, rows, dt) in want.items():
        w = W[name]
        sh = w.shape
        got = (sh.batch, sh.prompt_len, sh.resp_len, sh.n_heads, sh.n_kv_heads, sh.head_dim)
        assert (got, w.layers, w.steps, w.redraws_per_step, w.radius_k, w.max_age, w.vocab, w.logits_rows,
                w.logits_dtype) == (shape, layers, steps, redraws, K, max_age, vocab, rows, dt), name
    # 26 of 512 is 5 % rounded to the nearest position
    assert round(0.05 * 512) == W["traj32"].redraws_per_step == W["gqa_long"].redraws_per_step


def test_mask_state_rate_and_tokens_uniform():
    m = synth.mask_state(64, 4096, seed=3)
    assert abs(m.mean() - 0.5) < 0.01
    g = synth.tokens(64, 4096, 16, seed=3, mask=m)
    assert np.all(g[m == 1] == synth.MASK_TOKEN)
    counts = np.bincount(g[m == 0], minlength=16)
    assert counts.min() > 0.9 * counts.mean() and counts.max() < 1.1 * counts.mean()


def test_redraws_are_uniform_over_positions_and_other_tokens():
    # positions: each of G = 64 picked with probability n / G = 8 / 64
    hits = np.zeros(64)
    for step in range(2000):
        hits[synth.redraw_positions(7, step, 0, 64, 8)] += 1
    assert abs(hits.mean() / 2000 - 8 / 64) < 1e-12
    assert hits.min() > 0.85 * hits.mean() and hits.max() < 1.15 * hits.mean()
    # tokens: uniform over the 9 ids other than the current one
    cur = np.full(20000, 4, dtype=np.int32)
    new = synth.redraw_tokens(7, 0, 0, cur, 10)
    c = np.bincount(new, minlength=10)
    assert c[4] == 0
    others = np.delete(c, 4)
    assert others.min() > 0.9 * others.mean() and others.max() < 1.1 * others.mean()


def test_planted_token_boost_is_uniform_up_to_its_maximum():
    # the planted entry of a row is N(0, std^2) + U(0, boost): with std -> 0
    # (std 1e-6) the row maximum is that boost, uniform on [0, boost_max)
    z = synth.logits(20000, 64, seed=2, std=1e-6, boost_max=6.0, dtype="f32").astype(np.float64)
    top = z.max(axis=1)
    assert top.max() < 6.0 and top.min() >= 0.0
    assert abs(top.mean() - 3.0) < 0.05 and abs(top.std() - 6.0 / np.sqrt(12.0)) < 0.05
    # the planted id is uniform over the vocabulary
    c = np.bincount(z.argmax(axis=1), minlength=64)
    assert c.min() > 0.75 * c.mean() and c.max() < 1.25 * c.mean()
