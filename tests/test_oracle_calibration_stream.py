"""Section 5.3's online calibration inside the streaming loop (the oracle's side): between windows,
every decoding instance reports one pure-decode forward of a synthetic engine, and the scheduler
feeds these samples to its per-segment EMA factors before it scores the next window.

The synthetic engine runs each decode-batch segment slower than the profile by a fixed factor c_s
(c = 1.25 below batch 16, 1.6 from 16 up); its forward time at batch B and context S is
c_s ((b0 + b1 B) + b2 S), computed here in float64.  Every sample's ratio is then c_s up to one
rounding, so after k samples of segment s its factor is c_s - (c_s - 1) 0.98^k, whatever the
order of windows and instances.  The instances' KV capacity is 2^16 blocks (about 1M tokens),
so the stream keeps admitting requests; eviction keeps 3000 blocks cached per instance.

Pins:
- the closed form of every segment's factor after a six-window stream (the samples reach the
  segment of their batch size, and the factors persist across windows);
- a scheduler calibrated online scores a window bit for bit like a fresh one configured with the
  same factors (the calibration acts on the predictions through the factor table only);
- factors >= 1 only raise predicted TPOT, so the admitted set T of every request under the
  calibrated factors is a subset of T under factors 1 (same state, same caches).
"""
import numpy as np

import workload as W
from oracle import Oracle

SEG_LO = [0, 16]
SLOW = [1.25, 1.6]
MODEL = dict(W.MODEL_DEFAULT, seg_lo=SEG_LO, ema_factor=[1.0, 1.0])


def _engine_samples(st, model):
    """One decode forward per decoding instance: batch b, context S, the engine's time."""
    live = np.nonzero(st["b"] > 0)[0]
    B = st["b"][live].astype(np.int64)
    S = st["S"][live].astype(np.int64)
    seg = np.where(B >= SEG_LO[1], 1, 0)
    base = (float(model["b0"]) + float(model["b1"]) * B) + float(model["b2"]) * S
    t = (base * np.asarray(SLOW)[seg]).astype(np.float32)
    return B.astype(np.int32), S, t, seg


def _stream(windows=6, calibrate=True):
    wl = W.generate(0, seed=7, cap_blocks=1 << 16)
    ins = wl.instances
    o = Oracle(ins.I, MODEL, track_lru=True).load(ins)
    o.set_capacity(np.full(ins.I, 3000, np.uint64))
    req = wl.initial_requests()
    o.load_requests(req)
    counts = np.zeros(2, np.int64)
    for w in range(windows):
        win = wl.window if w == 0 else wl.next_window(24)
        o.schedule(win, window_id=w + 1, streaming=True)
        o.advance(20.0, 1000)
        if calibrate:
            B, S, t, seg = _engine_samples(o.get_state(), MODEL)
            o.calibrate(B, S, t, weight=0.02)
            counts += np.bincount(seg, minlength=2)
    return wl, o, counts


def test_factors_follow_the_closed_form_across_windows():
    _, o, k = _stream()
    assert k[0] > 0 and k[1] > 0, k  # both segments see samples
    want = np.asarray(SLOW) - (np.asarray(SLOW) - 1.0) * 0.98 ** k
    assert np.allclose(o.ema_factors(), want, rtol=1e-5), (o.ema_factors(), want, k)


def _fresh(state, factors, wl):
    o = Oracle(wl.instances.I, dict(MODEL, ema_factor=[float(f) for f in factors])).load(wl.instances)
    o.set_state(state["b"], state["qr"], state["q"], state["S"], state["M_KV"], state["B_max"])
    return o


def test_online_factors_act_like_configured_factors():
    """A window of fresh sessions (no cached prefix anywhere, so the caches play no part): the
    stream's scheduler and a fresh one with its state and factors agree bit for bit."""
    wl, o, _ = _stream()
    st, f = o.get_state(), o.ema_factors()
    probe = wl.next_window(32)
    rng = np.random.default_rng(3)
    probe.chain_hash = rng.integers(2, 2 ** 63, probe.chain_hash.shape[0], dtype=np.int64).astype(np.uint64)
    probe.tpot_target = np.linspace(120.0, 240.0, probe.R).astype(np.float32)
    a = o.score_rows(probe)
    b = _fresh(st, f, wl).score_rows(probe)
    assert np.array_equal(a["hits"], np.zeros_like(a["hits"]))
    assert np.any(a["cls"] == 0) and np.any(a["cls"] == 1)
    for key in ("cls", "best", "path"):
        assert np.array_equal(a[key], b[key]), key
    for key in ("tpot", "ttft"):
        assert np.array_equal(a[key].view(np.uint32), b[key].view(np.uint32)), key


def test_factors_above_one_shrink_the_admitted_set():
    wl, o, _ = _stream()
    st, f = o.get_state(), o.ema_factors()
    assert np.all(f > 1.0)
    win = wl.next_window(48)
    # the queued-prefill term puts predicted TPOT at 120-220 ms here: spread the targets over it
    win.tpot_target = np.linspace(120.0, 240.0, win.R).astype(np.float32)
    cal = _fresh(st, f, wl).score_rows(win)
    one = _fresh(st, [1.0, 1.0], wl).score_rows(win)
    assert np.array_equal(cal["hits"], one["hits"])
    in_T_cal, in_T_one = cal["cls"] == 0, one["cls"] == 0
    assert not np.any(in_T_cal & ~in_T_one)
    assert in_T_cal.sum() < in_T_one.sum()
    assert np.all(cal["tpot"][in_T_one] >= one["tpot"][in_T_one])
    assert np.any(cal["tpot"][in_T_one] > one["tpot"][in_T_one])
