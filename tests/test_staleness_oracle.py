"""Eq. theory-radius-bound on a layer with a known-Lipschitz prompt-cache map:
the cached step's error is zero at D_t = 0, below Gamma sqrt(D_t) for every
D_t, and grows with D_t; the radius K caps it at Gamma sqrt(K - 1)."""
import math

import numpy as np
import pytest

from oracle import staleness as S
from paper_2608_08086_gb300 import synth

SHAPE = synth.AttnShape(2, 96, 48, 4, 2, 64)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_error_below_gamma_sqrt_d(seed):
    ds = [0, 1, 2, 4, 8, 16, 32, 48]
    pts = S.curve(SHAPE, ds, seed=seed)
    assert pts[0][1] == 0.0
    for d, err, bound in pts:
        assert err <= bound * (1 + 1e-12), (d, err, bound)
    assert pts[-1][1] > 0


def test_radius_caps_every_cached_step():
    # a cached step happens only while D_t < K: every such error <= Gamma sqrt(K - 1)
    K = 9
    pts = S.curve(SHAPE, list(range(K)), seed=3)
    cap = pts[-1][2] / math.sqrt(K - 1)      # Gamma
    assert max(e for _, e, _ in pts) <= cap * math.sqrt(K - 1)


def test_gamma_matches_finite_difference_on_one_key():
    # a one-token change moves every prompt K/V row by alpha_j (A e' - A e): the
    # measured error sits under Gamma and above zero
    d, err, bound = S.curve(SHAPE, [1], seed=4)[0]
    assert 0 < err <= bound


def test_error_grows_with_the_drift():
    # nested drifts (D changes the first D positions of one order): averaged
    # over sequences of seeds, a larger distance gives a larger error
    ds = [2, 8, 48]
    errs = np.mean([[e for _, e, _ in S.curve(SHAPE, ds, seed=s)] for s in range(6)], axis=0)
    assert errs[0] < errs[1] < errs[2]


def test_error_scales_like_sqrt_d():
    # Eq. theory-radius-bound has the shape Gamma sqrt(D_t); with independent
    # drift directions the measured error follows it: err / sqrt(D) averaged
    # over seeds stays within a factor 1.5 from D = 1 to D = 48
    ds = [1, 4, 16, 48]
    errs = np.mean([[e for _, e, _ in S.curve(SHAPE, ds, seed=s)] for s in range(6)], axis=0)
    r = errs / np.sqrt(ds)
    assert r.max() < 1.5 * r.min()


def test_gamma_closed_form():
    # pieces whose norms are known by hand: embedding diameter 2 ([1, 0] to
    # [-1, 0]), largest alpha row norm 5 ([3, 4]), ||A_K||_2 = 2, ||A_V||_2 = 3
    # (diagonal), max ||q_i||_2 = 2, max |v| = 4 (response V), s = 1/4:
    # Gamma = 2 * 5 * (3 + 0.25 * 2 * 2 * 4) = 70
    model = {"emb": np.array([[1.0, 0.0], [0.0, 1.0], [-1.0, 0.0]]),
             "alpha": np.array([[3.0, 4.0], [0.0, 1.0]]),
             "a_k": np.diag([2.0, 1.0]), "a_v": np.diag([0.5, 3.0])}
    q = np.array([[[0.6, 0.8]], [[0.0, 2.0]]])
    v_cache = np.array([[1.5, -1.0]])
    v_resp = np.array([[-4.0, 0.5]])
    assert S.gamma(model, q, v_cache, v_resp, 0.25) == pytest.approx(70.0, rel=1e-14)


def test_reported_bound_grows_like_sqrt_d():
    # the bound the curve reports is Gamma sqrt(D_t) (Eq. theory-radius-bound):
    # zero at D = 0, and its ratios between distances are those of sqrt(D)
    ds = [0, 1, 4, 9, 25]
    pts = S.curve(SHAPE, ds, seed=5)
    assert pts[0][2] == 0.0
    for d, _, bound in pts[1:]:
        assert bound / pts[1][2] == pytest.approx(math.sqrt(d), rel=1e-12)
