"""The recompute-budget sweep (paper_2609_33224_gb300/diagnostics.py; Section 8's sensitivity study
of eta, Fig. 10 (a)-(b)) on the CPU: its per-window statistics on a hand-made scheduling, and the
sweep driven through a stand-in scheduler built on the oracle, checked against what Eq. 8 fixes:
- C grows with eta: a pair in C at eta is in C at every larger eta (so mean |C| never falls);
- at eta = 0, C is the set of capacity-eligible instances of least recompute W, which under the
  workload's coefficients (W = n (a1 + a2 L), increasing in n) are those with the longest hit;
- at a very large eta, C is all of A.
On the GPU the sweep makes the same two calls through the library (ps_set_model, then
ps_schedule_window with scores)."""
import numpy as np
import pytest

import workload as W
from oracle import Oracle
from paper_2609_33224_gb300.diagnostics import PAPER_ETAS, eta_sweep, window_stats


def test_window_stats_by_hand():
    """Three requests on four instances.  Row 0: C = {0, 1}, T = {0}; row 1: C = {2}, T = {};
    row 2: nothing in A.  Decisions: row 0 packed with a 10-block hit of its 320 tokens, row 1
    fallback with 2 blocks of 96 tokens, row 2 rejected."""
    cls = np.array([[0, 1, 2, 3], [3, 2, 1, 3], [3, 3, 3, 3]], np.uint8)
    st = window_stats(cls, np.array([0, 1, 2], np.uint8), np.array([10, 2, 0], np.uint32),
                      np.array([320, 96, 5000], np.uint32))
    assert st["requests"] == 3
    assert st["mean_C"] == 1.5 and st["mean_T"] == 0.5
    assert (st["packed"], st["fallback"], st["rejected"]) == (1, 1, 1)
    assert (st["cached_tokens"], st["admitted_tokens"]) == (16 * 12, 416)
    assert st["hit_rate"] == 16 * 12 / 416


def test_window_stats_of_an_empty_window():
    st = window_stats(np.zeros((0, 4), np.uint8), np.zeros(0, np.uint8), np.zeros(0, np.uint32),
                      np.zeros(0, np.uint32))
    assert st["requests"] == 0 and st["mean_C"] == 0.0 and st["hit_rate"] == 0.0


class OracleScheduler:
    """The two scheduler methods the sweep uses, on a fresh oracle per model (test stand-in)."""

    def __init__(self, wl, model):
        self.wl, self.model, self.calls = wl, dict(model), []

    def set_model(self, model):
        self.model = dict(model)

    def schedule_window(self, window, scores=()):
        o = Oracle(self.wl.instances.I, self.model).load(self.wl.instances)
        s = o.score_rows(window)  # no state change
        d = o.schedule(window)
        self.calls.append(dict(eta=self.model["eta"], cls=s["cls"], hits=s["hits"]))
        return dict(assign=d["assign"], path=d["path"], hit_chosen=d["hit_chosen"],
                    scores={"cls": s["cls"]} if "cls" in scores else {})


@pytest.mark.parametrize("config,rows", [(0, None), (1, 256)])
def test_sweep_against_eq8(config, rows):
    wl = W.generate(config)
    win = wl.window if rows is None else _head(wl.window, rows)
    sched = OracleScheduler(wl, wl.model)
    etas = PAPER_ETAS + (1e6,)
    res = eta_sweep(sched, win, wl.model, etas)
    assert [r["eta"] for r in res] == list(etas)
    assert sched.model == wl.model  # restored
    in_C = [c["cls"] <= 1 for c in sched.calls]
    for a, b in zip(in_C, in_C[1:]):
        assert not np.any(a & ~b)  # nested
    means = [r["mean_C"] for r in res]
    assert all(x <= y for x, y in zip(means, means[1:]))
    assert means[-1] > means[0]
    in_A = sched.calls[0]["cls"] <= 2
    assert np.array_equal(in_C[-1], in_A)  # eta huge: C = A
    h = sched.calls[0]["hits"].astype(np.int64)
    hmax = np.where(in_A, h, -1).max(axis=1, keepdims=True)
    assert np.array_equal(in_C[0], in_A & (h == hmax))  # eta 0: the longest hits in A
    for r in res:
        assert 0.0 <= r["hit_rate"] <= 1.0
        assert r["packed"] + r["fallback"] + r["rejected"] == win.R


def _head(win, n):
    """The first n requests of a window."""
    off = win.chain_off[: n + 1]
    return W.Window(chain_off=off.copy(), chain_hash=win.chain_hash[: int(off[-1])].copy(),
                    prompt_tokens=win.prompt_tokens[:n].copy(), ttft_target=win.ttft_target[:n].copy(),
                    tpot_target=win.tpot_target[:n].copy(), session=win.session[:n].copy(),
                    out_tokens=win.out_tokens[:n].copy())


def test_sweep_rejects_a_negative_eta_and_restores_the_model():
    wl = W.generate(0)
    sched = OracleScheduler(wl, wl.model)
    with pytest.raises(ValueError):
        eta_sweep(sched, wl.window, wl.model, (0.5, -1.0))
    assert sched.model == wl.model
