"""A second characterisation of the greedy (Algorithm 1 per request in arrival order, Section 4's
state tracking), used as a pin of the oracle's greedy: each decision can be reached from row s's
scores on the state before decision s - d, corrected only at the instances that decisions
s - d .. s - 1 picked.

Why it holds.  Between the two states, only the picked instances change: their queue and KV state,
and their caches (in-window inserts, which only lengthen hits).  Every other instance keeps its
capacity eligibility (A), its SLO admission (T) and its packing key; only W_min (Eq. 8) can move
its membership of C.  A picked instance can only lower W_min (a longer hit means fewer tokens to
recompute), so unless the instance holding W_min left A, the other instances can only leave C.
The instances outside the d + 1 smallest speculative keys keep keys at least the list's last one.
Hence the minimum over the list entries still in C, outside the picked set, and the picked
instances' true keys is the decision, whenever it is below the list's last key (or the list held
every candidate).

Keys follow Algorithm 1's order: in T by (-b, -h, qr, i), else (the fallback over C) by
((q + n)(b + qr + 1), i); Reject when A is empty.
"""
import numpy as np
import pytest

import workload as W
from oracle import Oracle


def _keys(cls, hits, st, L):
    out = {}
    for i in np.nonzero(cls <= 1)[0]:
        i = int(i)
        h, b, qr, q = int(hits[i]), int(st["b"][i]), int(st["qr"][i]), int(st["q"][i])
        n = L - 16 * h
        out[i] = (0, -b, -h, qr, i) if cls[i] == 0 else (1, (q + n) * (b + qr + 1), i)
    return out


def _longest_eligible_hit(cls, hits):
    a = cls <= 2
    return int(hits[a].max()) if a.any() else -1


def _head(win, n):
    off = win.chain_off[: n + 1]
    return W.Window(chain_off=off.copy(), chain_hash=win.chain_hash[: int(off[-1])].copy(),
                    prompt_tokens=win.prompt_tokens[:n].copy(), ttft_target=win.ttft_target[:n].copy(),
                    tpot_target=win.tpot_target[:n].copy(), session=win.session[:n].copy(),
                    out_tokens=win.out_tokens[:n].copy())


def _load(wl, flat_b):
    ins = wl.instances
    o = Oracle(ins.I, wl.model).load(ins)
    if flat_b:  # every instance decodes the same batch: D ties, so C and then Q decide in T
        o.set_state(np.full(ins.I, 20, np.int32), ins.qr, ins.q, ins.S, ins.M_KV, ins.B_max)
    return o


@pytest.mark.parametrize("config,rows,tpot,flat_b", [(0, 64, None, False), (1, 300, None, False),
                                                     (1, 300, 80.0, False), (1, 300, 80.0, True)])
def test_decisions_follow_from_lagged_scores(config, rows, tpot, flat_b):
    wl = W.generate(config)
    win = _head(wl.window, rows)
    if tpot is not None:
        win.tpot_target[:] = tpot  # more requests packed (class 0) than under the 50-ms target
    ins = wl.instances
    want = _load(wl, flat_b).schedule(win)
    rep = _load(wl, flat_b)
    lags = (1, 2, 8)
    spec, picks = {}, []
    fast = {d: 0 for d in lags}
    for s in range(win.R):
        ask = [s] + [s + d for d in lags if s + d < win.R]
        ev = rep.score_rows(win, rows=ask)
        st = rep.get_state()
        cls, hits = ev["cls"][0], ev["hits"][0]
        L = int(win.prompt_tokens[s])
        true_keys = _keys(cls, hits, st, L)
        best = int(ev["best"][0])
        # the greedy's decision is Algorithm 1 on the current state ...
        assert best == int(want["assign"][s])
        # ... and the smallest key of that state (Reject when nothing is in C)
        assert best == (min(true_keys.values())[-1] if true_keys else -1)
        for k, t in enumerate(ask[1:], start=1):
            Lt = int(win.prompt_tokens[t])
            spec[(t, t - s)] = (ev["cls"][k].copy(), ev["hits"][k].copy(), _keys(ev["cls"][k], ev["hits"][k], st, Lt))
        for d in lags:
            got = spec.pop((s, d), None)
            if got is None:
                continue
            scls, shits, skeys = got
            if _longest_eligible_hit(cls, hits) < _longest_eligible_hit(scls, shits):
                continue  # W_min rose: the full pass decides
            touched = {j for j in picks[s - d:s] if j >= 0}
            # untouched instances keep their class or leave C, never the other way
            for i in range(ins.I):
                if i not in touched and scls[i] != cls[i]:
                    assert scls[i] <= 1 and cls[i] == 2, (s, d, i, scls[i], cls[i])
            lst = sorted(skeys.values())[: d + 1]
            held_all = len(skeys) <= d + 1
            cand = [k for k in lst if k[-1] not in touched and cls[k[-1]] == scls[k[-1]]]
            cand += [true_keys[j] for j in touched if j in true_keys]
            pick = min(cand) if cand else None
            if held_all or (pick is not None and pick < lst[-1]):
                assert (pick[-1] if pick is not None else -1) == best, (s, d)
                fast[d] += 1
        # apply decision s: the picked instance queues the request and caches its chain
        if best >= 0:
            h = int(hits[best])
            st["qr"][best] += 1
            st["q"][best] += L - 16 * h
            st["S"][best] += L
            rep.set_state(st["b"], st["qr"], st["q"], st["S"], st["M_KV"], st["B_max"])
            ch = win.chain_hash[win.chain_off[s]:win.chain_off[s + 1]]
            rep.insert_chain(best, ch[h:], parent=int(ch[h - 1]) if h else 0)
        picks.append(best)
    for d in lags:
        assert fast[d] >= 0.8 * (win.R - d), (d, fast[d], win.R)
