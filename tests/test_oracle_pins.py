"""Pins for the oracle: facts fixed by the paper or by mathematics, not by the oracle itself.

  * hit length   -- brute-force token longest-common-prefix (Section 7 prefix tree) and the
                    "longest fully cached prefix" definition on non-closed sets;
  * latencies    -- hand-worked literals (tests/golden/hand_example.json), closed forms under the
                    workload coefficients (Eq. 6: W = n(a1 + a2 L), Z = L(a1 + a2 L));
  * filters      -- Section 6.1 special cases (eta = 0, Z = 0), Alg. 1 reject and fallback rules;
  * selection    -- D-C-Q order and LMetric fallback through the hand example, invariants;
  * greedy       -- hand-traced window, replay invariant.
"""
import numpy as np
import pytest

import workload as W
from oracle import Oracle
from tests.helpers import hand_example, lcp, make_window, seq_tokens

REL = 2e-6  # fp32 result vs a hand-computed decimal (a few roundings of 2^-24)


def _oracle(model, ins):
    return Oracle(ins.I, model).load(ins)


def _close(got, want, rel=REL):
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    assert np.all(np.abs(got - want) <= rel * np.abs(want) + 1e-9), (got, want)


# ---------------------------------------------------------------- hit length ---------------------
def test_hit_equals_token_lcp_bruteforce():
    """hit(r, i) = max over sequences s cached on i of floor(LCP_tokens(r, s) / 16)."""
    rng = np.random.default_rng(7)
    base = [rng.integers(0, 1 << 17, 900).astype(np.uint32) for _ in range(3)]
    seqs = []
    for b in base:
        for _ in range(4):  # branches diverging at arbitrary token positions
            cut = int(rng.integers(0, 800))
            tail = rng.integers(0, 1 << 17, int(rng.integers(0, 400))).astype(np.uint32)
            seqs.append(np.concatenate([b[:cut], tail]))
        seqs.append(b[: int(rng.integers(0, 900))])
    I = 5
    model = dict(W.MODEL_DEFAULT)
    o = Oracle(I, model)
    cached = {i: [] for i in range(I)}
    for k, s in enumerate(seqs):
        for i in range(I):
            if (k + i) % 3 == 0:
                o.insert_chain(i, W.chain_from_tokens(s))
                cached[i].append(s)
    queries = seqs + [b[: int(rng.integers(0, 900))] for b in base] + [np.zeros(0, np.uint32),
                                                                      base[0][:15], base[1][:16]]
    for qy in queries:
        ch = W.chain_from_tokens(qy)
        for i in range(I):
            want = max([lcp(qy, s) // 16 for s in cached[i]] + [0])
            assert o.hit(i, ch) == want


def test_hit_is_longest_fully_cached_prefix_on_gapped_set():
    """A set that is not prefix-closed: the hit stops at the first missing block."""
    ch = W.chain_from_tokens(seq_tokens("A", 16 * 40))
    o = Oracle(1, dict(W.MODEL_DEFAULT))
    o.insert_chain(0, ch[:3])
    o.insert_chain(0, ch[5:30], parent=int(ch[4]))
    assert o.hit(0, ch) == 3
    o.insert_chain(0, ch[3:4], parent=int(ch[2]))
    assert o.hit(0, ch) == 4
    o.insert_chain(0, ch[4:5], parent=int(ch[3]))
    assert o.hit(0, ch) == 30
    assert o.hit(0, ch[:0]) == 0


def test_hit_bounded_and_monotone_under_superset():
    wl = W.generate(0)
    win, ins = wl.window, wl.instances
    o = _oracle(wl.model, ins)
    rows = o.score_rows(win)["hits"]
    nb = np.diff(win.chain_off).astype(np.int64)
    assert np.all(rows <= nb[:, None])
    # add every window chain to instance 0: hits there can only grow, to the full chain
    for r in range(win.R):
        o.insert_chain(0, win.chain_hash[win.chain_off[r]:win.chain_off[r + 1]])
    rows2 = o.score_rows(win)["hits"]
    assert np.all(rows2 >= rows)
    assert np.array_equal(rows2[:, 0], nb)


# ---------------------------------------------------------------- hand example -------------------
def test_hand_example_score_mode(hand):
    model, ins, win, d = hand
    out = _oracle(model, ins).score_rows(win)
    e = d["score_mode"]
    assert out["hits"].tolist() == e["hits"]
    assert out["cls"].tolist() == e["cls"]
    assert out["best"].tolist() == e["best"]
    assert out["path"].tolist() == e["path"]
    for r in range(win.R):
        if e["tpot"][r] is not None:
            _close(out["tpot"][r], e["tpot"][r])
            _close(out["ttft"][r], e["ttft"][r])


def test_hand_example_schedule_mode(hand):
    model, ins, win, d = hand
    o = _oracle(model, ins)
    out = o.schedule(win)
    e = d["schedule_mode"]
    assert out["assign"].tolist() == e["assign"]
    assert out["path"].tolist() == e["path"]
    assert out["hit_chosen"].tolist() == e["hit_chosen"]
    st = o.get_state()
    for i, f in enumerate(e["final_state"]):
        for k in ("b", "qr", "q", "S"):
            assert int(st[k][i]) == f[k], (i, k)


def test_paper_interference_form_hand_values(hand):
    """Eq. 9: decode term + [A > 0] T_pf(n, c) / max(1, L_out); hand values for request r0."""
    model, ins, win, d = hand
    m = dict(model, interference_mode=1)
    out = _oracle(m, ins).score_rows(win, rows=[0])
    # instance 0: 13.3258 + 10.66314/556; instance 1: 15.1758 + 21.56362/556 (qr = 0, b = 20 > 0)
    _close(out["tpot"][0][:2], [13.3258 + 10.66314 / 556, 15.1758 + 21.56362 / 556])
    # an instance with no active request pays no interference
    ins0 = W.Instances(**{k: getattr(ins, k).copy() for k in ins.__dataclass_fields__})
    ins0.b[1] = 0
    out0 = _oracle(m, ins0).score_rows(win, rows=[0])
    _close(out0["tpot"][0][1], 8 + 0.15 * 1 + 2e-5 * 201290)


def test_ema_segments_scale_decode_term_only(hand):
    """Section 5.3 online factor: scales the decode term of the projected batch's segment."""
    model, ins, win, d = hand
    m = dict(model, seg_lo=[0, 17, 33], ema_factor=[1.0, 1.5, 2.0])
    out = _oracle(m, ins).score_rows(win, rows=[0])
    # B = 22, 21, 33, 9 -> factors 1.5, 1.5, 2.0, 1.0
    _close(out["tpot"][0], [13.3258 * 1.5 + 5.064, 15.1758 * 1.5 + 3.112, 31.9758 * 2 + 24.648,
                            10.3758 + 8.04])


def test_ttft_filter_and_prefill_floor(hand):
    """A 1-ms TTFT target is floored at the cold prefill time T_pf(L, 0) = 32.4641 ms (r0)."""
    model, ins, win, d = hand
    tight = make_window([(seq_tokens("A", 1290), 1.0, 50.0)])
    out = _oracle(model, ins).score_rows(tight)
    # TTFT 35.66314 (instance 0) > 32.4641 >= 21.56362 (instance 1): only instance 1 is in T
    assert out["cls"][0].tolist() == [1, 0, 2, 3]
    assert out["best"].tolist() == [1]
    out_off = _oracle(dict(model, ttft_filter=0), ins).score_rows(tight)
    assert out_off["best"].tolist() == [0]


# ---------------------------------------------------------------- closed forms -------------------
def test_cold_instance_latencies_closed_form():
    """b = qr = q = S = 0, nothing cached: TPOT = 8.15 + 0.00402 L, TTFT = 5 + 0.02 L + 1e-6 L^2."""
    Ls = [16, 17, 1000, 4096, 65536 + 5, 131072]
    win = make_window([(seq_tokens("B", L), 3000.0, 50.0) for L in Ls])
    I = 2
    o = Oracle(I, dict(W.MODEL_DEFAULT))
    o.set_state(np.zeros(I, np.int32), np.zeros(I, np.int32), np.zeros(I, np.int64),
                np.zeros(I, np.int64), np.full(I, 10 ** 9, np.int64), np.full(I, 64, np.int32))
    out = o.score_rows(win)
    L = np.array(Ls, np.float64)
    _close(out["tpot"][:, 0], 8.15 + 0.00402 * L)
    _close(out["ttft"][:, 0], 5 + 0.02 * L + 1e-6 * L * L)
    assert np.all(out["hits"] == 0)


@pytest.mark.parametrize("cfg", [0, 1])
def test_rho_closed_form(cfg):
    """With a2 = a3 and a4 = a5 = 0, Eq. 8's rho equals (n - n_min) / L exactly in real
    arithmetic; eta = 0.5, so instance i leaves C iff 2 (n_i - n_min) > L."""
    wl = W.generate(cfg) if cfg == 0 else W.generate(1, window_requests=64)
    win, ins = wl.window, wl.instances
    o = _oracle(wl.model, ins)
    out = o.score_rows(win)
    L = win.prompt_tokens.astype(np.int64)
    n = L[:, None] - 16 * out["hits"].astype(np.int64)
    inA = out["cls"] != 3
    boundary = 0
    checked = 0
    for r in range(win.R):
        if not inA[r].any():
            continue
        nmin = n[r][inA[r]].min()
        lhs = 2 * (n[r] - nmin)
        for i in np.nonzero(inA[r])[0]:
            checked += 1
            if abs(int(lhs[i]) - int(L[r])) <= 2:
                boundary += 1
                continue
            assert (out["cls"][r, i] == 2) == (lhs[i] > L[r]), (r, i)
        # TTFT with an empty queue is T_pf(n, c) = a0 + n (a1 + a2 L)
    assert checked > 0
    assert boundary <= checked // 100
    qz = ins.qr == 0
    if qz.any():
        want = 5 + n[:, qz] * (0.02 + 1e-6 * L[:, None])
        _close(out["ttft"][:, qz], want, rel=4e-6)


# ---------------------------------------------------------------- special cases ------------------
def _flat_instances(I, b=10, qr=0, q=0, S=0, M=10 ** 9, bmax=64):
    return dict(b=np.full(I, b, np.int32), qr=np.full(I, qr, np.int32), q=np.full(I, q, np.int64),
                S=np.full(I, S, np.int64), M_KV=np.full(I, M, np.int64),
                B_max=np.full(I, bmax, np.int32))


def _graded_oracle(model, I=6, **kw):
    """Instance i caches the first 10 i blocks of sequence A."""
    o = Oracle(I, model)
    ch = W.chain_from_tokens(seq_tokens("A", 16 * 100))
    for i in range(I):
        o.insert_chain(i, ch[:10 * i])
    s = _flat_instances(I, **kw)
    o.set_state(s["b"], s["qr"], s["q"], s["S"], s["M_KV"], s["B_max"])
    return o


def test_eta_zero_keeps_only_min_cost():
    """Section 6.1: eta = 0 retains only the minimum-cost candidates."""
    o = _graded_oracle(dict(W.MODEL_DEFAULT, eta=0.0))
    out = o.score_rows(make_window([(seq_tokens("A", 1600), 3000.0, 50.0)]))
    assert out["cls"][0].tolist() == [2, 2, 2, 2, 2, 0]
    assert out["best"].tolist() == [5]


def test_eta_large_keeps_all_of_A():
    o = _graded_oracle(dict(W.MODEL_DEFAULT, eta=1.0))
    out = o.score_rows(make_window([(seq_tokens("A", 1600), 3000.0, 50.0)]))
    assert np.all(out["cls"][0] <= 1)


def test_zero_cache_benefit_keeps_all_of_A():
    """Section 6.1: if Z_r = 0 all capacity-eligible candidates remain (prefill cost flat)."""
    m = dict(W.MODEL_DEFAULT, a1=0.0, a2=0.0, a3=0.0, eta=0.0)
    o = _graded_oracle(m)
    out = o.score_rows(make_window([(seq_tokens("A", 1600), 3000.0, 50.0)]))
    assert np.all(out["cls"][0] <= 1)
    # equal decode batches; most cached blocks wins among T
    assert out["best"].tolist() == [5]


def test_capacity_guard_rejects_when_A_empty():
    """Alg. 1: no capacity-eligible instance -> Reject; slot limit and KV limit each suffice."""
    win = make_window([(seq_tokens("A", 1600), 3000.0, 50.0)])
    o = _graded_oracle(dict(W.MODEL_DEFAULT), b=63, qr=1, bmax=64)   # 63 + 1 + 1 > 64
    out = o.score_rows(win)
    assert out["best"].tolist() == [-1] and out["path"].tolist() == [2]
    assert np.all(out["cls"] == 3)
    o = _graded_oracle(dict(W.MODEL_DEFAULT), S=10 ** 6, M=10 ** 6 + 1599)  # S + L > M_KV
    assert o.score_rows(win)["best"].tolist() == [-1]
    o = _graded_oracle(dict(W.MODEL_DEFAULT), S=10 ** 6, M=10 ** 6 + 1600)  # S + L == M_KV fits
    assert o.score_rows(win)["best"].tolist() == [5]


def test_fallback_when_T_empty_prefers_cache_under_equal_load():
    """T empty -> CacheAwareLB over C: with identical load the most-cached candidate wins and the
    pick stays inside C (Alg. 1 fallback keeps the capacity and recompute constraints)."""
    o = _graded_oracle(dict(W.MODEL_DEFAULT))
    out = o.score_rows(make_window([(seq_tokens("A", 1600), 3000.0, 1.0)]))
    assert out["path"].tolist() == [1]
    assert out["best"].tolist() == [5]
    assert out["cls"][0][5] == 1


def test_decode_batch_dominates_cache_in_T():
    """D before C (Section 6.2): a packed pick never has fewer decoding requests than any
    instance of T, and among equal decode batches never fewer cached blocks."""
    wl = W.generate(0)
    o = _oracle(wl.model, wl.instances)
    out = o.score_rows(wl.window)
    b = wl.instances.b
    for r in range(wl.window.R):
        T = np.nonzero(out["cls"][r] == 0)[0]
        if T.size == 0:
            continue
        j = out["best"][r]
        assert out["path"][r] == 0 and j in T
        assert b[j] == b[T].max()
        same = T[b[T] == b[j]]
        assert out["hits"][r, j] == out["hits"][r, same].max()


# ---------------------------------------------------------------- invariants ---------------------
@pytest.mark.parametrize("cfg", [0])
def test_score_invariants(cfg):
    wl = W.generate(cfg)
    win = wl.window
    o = _oracle(wl.model, wl.instances)
    out = o.score_rows(win)
    for r in range(win.R):
        cls = out["cls"][r]
        j = out["best"][r]
        anyA = (cls != 3).any()
        assert (j < 0) == (not anyA)                 # Reject iff A is empty
        if (cls == 0).any():                          # a feasible pick whenever T is non-empty
            assert out["path"][r] == 0 and cls[j] == 0
            assert out["tpot"][r, j] < win.tpot_target[r]
        elif anyA:
            assert out["path"][r] == 1 and cls[j] == 1


def test_greedy_replay_equals_single_request_rule():
    """Each greedy decision equals Algorithm 1 on the state left by all earlier decisions."""
    wl = W.generate(0)
    win, ins = wl.window, wl.instances
    o = _oracle(wl.model, ins)
    sched = o.schedule(win)
    replay = _oracle(wl.model, ins)
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
    assert (sched["path"] == 0).any()
