"""Pins for the oracle's policy variants: the admission/fallback ablations of Table 3 (G, C, T, CT,
F) and the instance orders of Table 4 (D, D-Q, D-C, D-Q-C, H-C-Q against the adopted D-C-Q),
worked by hand on one request against eight instances.

Request: L = 1600 tokens (100 blocks), TTFT target 1e6 ms.  Workload coefficients (a0 5, a1 0.02,
a2 = a3 = 1e-6; b0 8, b1 0.15, b2 2e-5, g_q 0.004; eta 0.5), q = S = 0 unless stated:
  Z = L (a1 + a2 L) = 34.56, eta Z = 17.28, W = n (a1 + a2 L) = 0.0216 n with n = 1600 - 16 h.
  The best hit is 90 blocks (n 160), so C holds the instances with n <= 160 + 800, i.e. h >= 40.
  TPOT = (8 + 0.15 B) + 2e-5 (S + L) + 0.004 (q + n), B = b + qr + 1.

  inst  b  qr      q   hit   n     B   TPOT (ms)   in C   LMetric (q + n) B
   0   10   2   2000    90   160   13   18.622      yes    28080
   1   12   3      0    45   880   16   13.952      yes    14080
   2   12   3      0    60   640   16   12.992      yes    10240
   3   12   1      0    45   880   14   13.652      yes    12320
   4   12   2      0    60   640   15   12.842      yes     9600
   5   12   1      0    50   800   14   13.332      yes    11200
   6   20   0      0     0  1600   21   17.582      no         -
   7   40   0  20000    90   160   41   94.822      yes   826560
"""
import numpy as np
import pytest

import workload as W
from oracle import ABLATIONS, SELECTORS, Oracle
from tests.helpers import make_window, seq_tokens

TOKENS = seq_tokens("A", 1600)
STATE = dict(b=[10, 12, 12, 12, 12, 12, 20, 40], qr=[2, 3, 3, 1, 2, 1, 0, 0],
             q=[2000, 0, 0, 0, 0, 0, 0, 20000], hit=[90, 45, 60, 45, 60, 50, 0, 90])


def _pick(tpot_target, **policy):
    model = dict(W.MODEL_DEFAULT, **policy)
    o = Oracle(8, model)
    chain = W.chain_from_tokens(TOKENS)
    for i, h in enumerate(STATE["hit"]):
        if h:
            o.insert_chain(i, chain[:h])
    o.set_state(np.array(STATE["b"], np.int32), np.array(STATE["qr"], np.int32), np.array(STATE["q"], np.int64),
                np.zeros(8, np.int64), np.full(8, 10 ** 9, np.int64), np.full(8, 1000, np.int32))
    r = o.score_rows(make_window([(TOKENS, 1e6, tpot_target)]))
    assert list(r["hits"][0]) == STATE["hit"]
    return int(r["best"][0]), int(r["path"][0]), r


def test_hand_table_latencies_and_cache_filter():
    _, _, r = _pick(50.0)
    want = [18.622, 13.952, 12.992, 13.652, 12.842, 13.332, 17.582, 94.822]
    assert np.allclose(r["tpot"][0], want, rtol=2e-6)
    # classes: 0 in T, 1 in C outside T, 2 in A outside C
    assert list(r["cls"][0]) == [0, 0, 0, 0, 0, 0, 2, 1]


@pytest.mark.parametrize("name,want", [("D-C-Q", 4), ("D", 1), ("D-Q", 3), ("D-C", 2), ("D-Q-C", 5),
                                       ("H-C-Q", 0)])
def test_selectors_inside_T(name, want):
    """Inside T = {0..5}: D keeps b = 12 (1..5); D-Q the fewest queued (3, 5); D-C the most cached
    (2, 4); D-C-Q then the fewest queued (4); D-Q-C then the most cached (5); H the smallest
    headroom 50 - TPOT, instance 0's 31.378 ms.  The lowest id breaks what remains."""
    best, path, _ = _pick(50.0, selector=SELECTORS[name])
    assert (best, path) == (want, 0)


@pytest.mark.parametrize("name,want", [("F", 4), ("CT", 4), ("C", 7), ("G", 7), ("T", 6)])
def test_ablations_with_T_non_empty(name, want):
    """G: capacity only, every instance admissible, the most decoding (7).  C: the cache filter only,
    instance 7 (in C, TPOT over target) is admissible.  T: TPOT only, C = A, instance 6 (b 20) is
    admissible and 7 is not.  CT and F: the adopted sets, D-C-Q picks 4."""
    best, path, _ = _pick(50.0, **ABLATIONS[name])
    assert (best, path) == (want, 0)


@pytest.mark.parametrize("name,want", [("F", 4), ("CT", 7), ("T", 7)])
def test_fallbacks_with_T_empty(name, want):
    """A 5-ms TPOT target empties T.  F: cache-aware LB (LMetric) over C, the smallest (q + n) B is
    instance 4's 9600.  CT: D-C-Q over C, the most decoding is 7.  T: D-C-Q over C = A, again 7."""
    best, path, _ = _pick(5.0, **ABLATIONS[name])
    assert (best, path) == (want, 1)


def test_default_policy_is_algorithm_1():
    """The defaults are the F configuration with the D-C-Q order."""
    assert _pick(50.0)[:2] == _pick(50.0, **ABLATIONS["F"], selector=SELECTORS["D-C-Q"])[:2]
    assert _pick(5.0)[:2] == _pick(5.0, **ABLATIONS["F"])[:2]


@pytest.mark.parametrize("policy", [dict(ABLATIONS["G"]), dict(ABLATIONS["T"]), dict(ABLATIONS["CT"]),
                                    dict(selector=SELECTORS["H-C-Q"]), dict(selector=SELECTORS["D-Q-C"])])
def test_greedy_replay_under_policy_variants(policy):
    """Under every variant, each greedy decision equals the single-request rule on the state left by
    the earlier decisions (the greedy applies the variant, not the default)."""
    wl = W.generate(0)
    win, ins = wl.window, wl.instances
    model = dict(wl.model, **policy)
    sched = Oracle(ins.I, model).load(ins).schedule(win)
    replay = Oracle(ins.I, model).load(ins)
    for r in range(win.R):
        one = replay.score_rows(win, rows=[r])
        assert one["best"][0] == sched["assign"][r] and one["path"][0] == sched["path"][r]
        j = int(one["best"][0])
        if j < 0:
            continue
        h = int(one["hits"][0, j])
        st = replay.get_state()
        L = int(win.prompt_tokens[r])
        st["qr"][j] += 1
        st["q"][j] += L - 16 * h
        st["S"][j] += L
        replay.set_state(st["b"], st["qr"], st["q"], st["S"], st["M_KV"], st["B_max"])
        ch = win.chain_hash[win.chain_off[r]:win.chain_off[r + 1]]
        replay.insert_chain(j, ch[h:], parent=int(ch[h - 1]) if h else 0)
    if policy in (dict(ABLATIONS["G"]), dict(ABLATIONS["T"])):  # these admit other instances here
        default = Oracle(ins.I, wl.model).load(ins).schedule(win)
        assert not np.array_equal(sched["assign"], default["assign"])
