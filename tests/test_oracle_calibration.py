"""Pins for the oracle's online calibration (Section 5.3): one multiplicative EMA factor per
decode-batch segment, starting at 1, tracking the measured-to-predicted ratio of pure-decode
forwards with update weight 0.02, ratios clipped to [0.5, 2] and factors to [1, 2]; the factor of the
projected batch size scales the decode term of the TPOT prediction.

Workload coefficients: the base decode prediction is (8 + 0.15 B) + 2e-5 S."""
import numpy as np

import workload as W
from oracle import Oracle
from tests.helpers import make_window, seq_tokens

MODEL = dict(W.MODEL_DEFAULT, seg_lo=[0, 17], ema_factor=[1.0, 1.0])


def _oracle():
    o = Oracle(1, MODEL)
    o.set_state(np.array([20], np.int32), np.array([0], np.int32), np.array([0], np.int64),
                np.array([10000], np.int64), np.array([10 ** 9], np.int64), np.array([1000], np.int32))
    return o


def test_hand_trace_with_clipping_and_segments():
    """B = 20, S = 10000: base = 11 + 0.2 = 11.2 ms (segment 1, B >= 17).
    16.8 ms: ratio 1.5, f = 1 + 0.02 * 0.5 = 1.01.
    40 ms: ratio 3.57 clipped to 2, f = 1.01 + 0.02 * 0.99 = 1.0298.
    2 ms: ratio 0.18 clipped to 0.5, f = 1.0298 - 0.02 * 0.5298 = 1.019204.
    B = 5 (segment 0), 4.5 ms against base 8.75 + 0.2 = 8.95: ratio 0.503, f = 0.99 clipped to 1."""
    o = _oracle()
    o.calibrate([20], [10000], [16.8])
    assert np.isclose(o.ema_factors()[1], 1.01, rtol=1e-6)
    o.calibrate([20, 20], [10000, 10000], [40.0, 2.0])
    f = o.ema_factors()
    assert np.isclose(f[1], 1.019204, rtol=1e-6) and f[0] == 1.0
    o.calibrate([5], [10000], [4.5])
    assert o.ema_factors()[0] == 1.0


def test_closed_form_of_a_constant_ratio():
    """k samples of ratio r from f = 1: f_k = r - (r - 1) 0.98^k (real arithmetic)."""
    o = _oracle()
    k, r = 60, 1.6
    o.calibrate(np.full(k, 20), np.full(k, 10000), np.full(k, 11.2 * r, np.float32))
    assert np.isclose(o.ema_factors()[1], r - (r - 1) * 0.98 ** k, rtol=2e-5)


def test_factor_bounds():
    o = _oracle()
    o.calibrate(np.full(3000, 20), np.full(3000, 10000), np.full(3000, 1000.0, np.float32))
    f = o.ema_factors()[1]
    assert 1.99 < f <= 2.0
    o2 = _oracle()
    o2.calibrate(np.full(500, 20), np.full(500, 10000), np.full(500, 0.001, np.float32))
    assert o2.ema_factors()[1] == 1.0


def test_factor_scales_the_decode_term_of_tpot():
    """After calibration to f, a request of L = 160 tokens on the B = 21 instance predicts
    TPOT = ((8 + 0.15 * 21) + 2e-5 * 10160) f + 0.004 * 160."""
    o = _oracle()
    o.calibrate(np.full(40, 20), np.full(40, 10000), np.full(40, 11.2 * 1.5, np.float32))
    f = float(o.ema_factors()[1])
    r = o.score_rows(make_window([(seq_tokens("A", 160), 1e6, 1e6)]))
    dec = (8 + 0.15 * 21) + 2e-5 * 10160
    assert np.isclose(r["tpot"][0][0], dec * f + 0.004 * 160, rtol=3e-6)
