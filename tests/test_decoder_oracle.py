"""The synthetic rollback decoder (stand-in for D) on the oracle, against
hand-worked cases, and the closed-loop trajectory's invariants."""
import numpy as np

from oracle import oracle as O
from oracle import trajectory as OT
from paper_2608_08086_gb300 import synth

M = -1


def test_accept_remask_and_keep():
    g = np.array([[M, M, 7, 9, 3]], np.int32)
    mp = np.array([0.95, 0.50, 0.99, 0.2, 0.6])
    t1 = np.array([11, 12, 13, 14, 15])
    cp = np.array([0.0, 0.0, 0.04, 0.05, 0.9])      # masked rows carry 0
    g2, ch = O.decoder_update(g, mp, t1, cp, 0.9, 0.05, M)
    # pos 0 accepted (0.95 >= 0.9); pos 1 stays masked; pos 2 re-masked (0.04 < 0.05);
    # pos 3 kept (0.05 is not < 0.05); pos 4 kept
    np.testing.assert_array_equal(g2, [[11, M, M, 9, 3]])
    np.testing.assert_array_equal(ch, [[1, 0, 1, 0, 0]])


def test_progress_rule_takes_the_most_confident_masked_position():
    g = np.array([[M, 5, M, M], [1, 2, 3, 4]], np.int32)
    mp = np.array([0.3, 0.99, 0.7, 0.7, 0.9, 0.9, 0.9, 0.9])
    t1 = np.array([20, 21, 22, 23, 30, 31, 32, 33])
    cp = np.array([0.0, 0.5, 0.0, 0.0, 0.5, 0.5, 0.5, 0.5])
    g2, ch = O.decoder_update(g, mp, t1, cp, 0.9, 0.05, M)
    # sequence 0: nothing reaches 0.9 among masked; the tie 0.7 / 0.7 goes to the lower index 2
    np.testing.assert_array_equal(g2[0], [M, 5, 22, M])
    # sequence 1: nothing masked, nothing below 0.05: unchanged
    np.testing.assert_array_equal(g2[1], [1, 2, 3, 4])
    np.testing.assert_array_equal(ch, [[0, 0, 1, 0], [0, 0, 0, 0]])


def test_threshold_is_inclusive_for_accept():
    g = np.array([[M, M]], np.int32)
    g2, _ = O.decoder_update(g, np.array([0.9, 0.1]), np.array([4, 5]), np.zeros(2), 0.9, 0.05, M)
    np.testing.assert_array_equal(g2, [[4, M]])
    # two positions exactly at the threshold: both accepted (the progress rule
    # alone would take one)
    g2, ch = O.decoder_update(np.array([[M, M, M]], np.int32), np.array([0.9, 0.9, 0.3]), np.array([4, 5, 6]),
                              np.zeros(3), 0.9, 0.05, M)
    np.testing.assert_array_equal(g2, [[4, 5, M]])
    np.testing.assert_array_equal(ch, [[1, 1, 0]])


def test_closed_loop_trajectory_makes_progress_and_rolls_back():
    wl = synth.WORKLOADS["tiny"]
    recs = OT.run(wl, seed=0, decoder="closed", steps=10)
    masked = [(r["g"] == M).sum() for r in recs]
    assert masked[0] == wl.shape.resp_len and masked[-1] < masked[0] // 2
    # every step changes at least one position (the progress rule) until done
    assert all(r["changed"].sum() >= 1 for r in recs[1:])
    # some accepted token was rolled back (re-masked) along the way
    remasked = sum(int(((r0["g"] != M) & (r1["g"] == M)).sum()) for r0, r1 in zip(recs, recs[1:]))
    assert remasked > 0
    # the refresh rule saw the decoder's drift: distance = changed positions since the anchor
    tgt, _ = synth.closed_loop_targets(wl, 0)
    assert ((recs[-1]["g"] == tgt) | (recs[-1]["g"] == M)).mean() > 0.8
