"""Pins for the oracle's streaming rules (between windows): hand-traced engine progress and
leaf-first LRU eviction, plus the invariants they must keep."""
import numpy as np

import workload as W
from oracle import Oracle
from tests.helpers import make_window, seq_tokens


def _one_instance(model=None, cap=10 ** 6):
    o = Oracle(1, dict(model or W.MODEL_DEFAULT), track_lru=True)
    o.set_state(np.zeros(1, np.int32), np.zeros(1, np.int32), np.zeros(1, np.int64), np.zeros(1, np.int64),
                np.full(1, 10 ** 9, np.int64), np.full(1, 64, np.int32))
    o.set_capacity(np.array([cap], np.uint64))
    return o


def test_advance_hand_trace():
    """Two decoding requests (L 1000 out 10 rem 3; L 2000 out 50 rem 40) and two queued ones
    (L 500 out 5 prefill 700; L 800 out 7 prefill 600): S = 1007 + 2010 + 500 + 800 = 4317.
    Window 1: T_iter = 8 + 0.15*2 + 2e-5*4317 = 8.38634 ms -> k = floor(20 / 8.38634) = 2 tokens
    each (S 4321); the drain finishes the first queued request (700) and takes 300 of the second.
    Window 2: T_iter = 8 + 0.15*3 + 2e-5*4321 = 8.53642 -> k = 2; the first request emits its
    last token and leaves (S -= 1010), the others emit 2; the drain finishes the second queued
    request (300)."""
    o = _one_instance()
    o.load_requests(dict(inst=[0, 0, 0, 0], state=[1, 1, 0, 0], L=[1000, 2000, 500, 800], out=[10, 50, 5, 7],
                         rem=[3, 40, 700, 600]))
    st = o.get_state()
    assert (st["b"][0], st["qr"][0], st["q"][0], st["S"][0]) == (2, 2, 1300, 4317)
    o.advance(20.0, 1000)
    st = o.get_state()
    assert (st["b"][0], st["qr"][0], st["q"][0], st["S"][0]) == (3, 1, 300, 4321)
    o.advance(20.0, 1000)
    st = o.get_state()
    assert (st["b"][0], st["qr"][0], st["q"][0], st["S"][0]) == (3, 0, 0, 4326 - 1010)


def test_advance_slow_iteration_still_emits_one_token():
    """k = max(1, floor(window / T_iter)): a 100-ms iteration still advances each request by one."""
    o = _one_instance(dict(W.MODEL_DEFAULT, b0=100.0))
    o.load_requests(dict(inst=[0], state=[1], L=[100], out=[3], rem=[2]))
    o.advance(20.0, 1000)
    assert o.get_state()["S"][0] == 100 + 1 + 1
    o.advance(20.0, 1000)
    st = o.get_state()
    assert (st["b"][0], st["S"][0]) == (0, 0)


def test_leaf_first_lru_eviction_hand_trace():
    """Capacity 5 with chain A (5 blocks, last_use 1) and chain B (3 blocks, last_use 2): the three
    evictions take A's leaf three times (A4, A3, A2), never B's more recent leaf."""
    A = W.chain_from_tokens(seq_tokens("A", 16 * 5))
    B = W.chain_from_tokens(seq_tokens("B", 16 * 3))
    o = _one_instance(cap=5)
    o.insert_chain(0, A, last_use=1)
    o.insert_chain(0, B, last_use=2)
    assert o.cached_blocks(0) == 8
    o.advance(20.0, 0)
    assert o.cached_blocks(0) == 5
    assert [o.contains(0, int(h)) for h in A] == [True, True, False, False, False]
    assert all(o.contains(0, int(h)) for h in B)


def test_eviction_order_breaks_last_use_ties_by_hash_and_touch_protects_prefix():
    """Equal last_use: the smaller block hash goes first.  Scheduling a request stamps its whole
    cached prefix, so the other chain's leaves go first."""
    A = W.chain_from_tokens(seq_tokens("A", 16 * 4))
    B = W.chain_from_tokens(seq_tokens("B", 16 * 4))
    o = _one_instance(cap=7)
    o.insert_chain(0, A, last_use=3)
    o.insert_chain(0, B, last_use=3)
    o.advance(20.0, 0)
    first = min(int(A[-1]), int(B[-1]))
    assert not o.contains(0, first) and o.cached_blocks(0) == 7
    o2 = _one_instance(cap=6)
    o2.insert_chain(0, A, last_use=3)
    o2.insert_chain(0, B, last_use=3)
    o2.schedule(make_window([(seq_tokens("A", 16 * 4), 3000.0, 1000.0)]), window_id=9)
    assert o2.last_use(0, int(A[0])) == 9 and o2.last_use(0, int(A[-1])) == 9
    o2.advance(20.0, 0)
    assert all(o2.contains(0, int(h)) for h in A)
    assert [o2.contains(0, int(h)) for h in B] == [True, True, False, False]


def test_streaming_invariants_on_a_small_stream():
    """Prefix closure after eviction, caches at or under capacity, state consistent with the queues."""
    wl = W.generate(0, seed=5)
    ins = wl.instances
    cap = np.full(ins.I, 3000, np.uint64)
    o = Oracle(ins.I, wl.model, track_lru=True).load(ins)
    o.set_capacity(cap)
    o.load_requests(dict(inst=[], state=[], L=[], out=[], rem=[]))
    st0 = o.get_state()
    assert np.all(st0["b"] == 0) and np.all(st0["S"] == 0)
    admitted = 0
    for w in range(6):
        win = wl.window if w == 0 else wl.next_window(24)
        d = o.schedule(win, window_id=w + 1, streaming=True)
        admitted += int((d["path"] < 2).sum())
        st = o.get_state()
        assert np.all(st["q"] >= 0) and np.all(st["qr"] >= 0)
        o.advance(20.0, 1000)
        for i in range(ins.I):
            assert o.cached_blocks(i) <= 3000
        # closure: every cached block of every window chain is preceded by a cached parent
        for r in range(win.R):
            ch = win.chain_hash[win.chain_off[r]:win.chain_off[r + 1]]
            for i in range(ins.I):
                present = [o.contains(i, int(h)) for h in ch]
                k = present.index(False) if False in present else len(present)
                assert not any(present[k:]), (w, r, i)
    assert admitted > 0
