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
