"""Windows in the shared-prefix form (ps_window.parent) on the GPU, through the C ABI.

The library rebuilds every chain on the device from the requests' own blocks and parent links, so a
window sent in this form must score and schedule exactly as the same window sent whole: against the
oracle on the tiny and eval-scale windows, against the stored oracle run on the production window
(every pick, every score chunk's digest, every greedy decision and the pending state), and through a
few carried streaming windows.  Malformed links are refused before any work.
"""
import numpy as np
import pytest

import workload as W
from oracle import Oracle
from tests.golden import make_fullsize as G

pytestmark = pytest.mark.gpu

WANT = ("hits", "tpot", "ttft", "cls", "best", "path")


@pytest.fixture(scope="module")
def P():
    import torch
    if not torch.cuda.is_available():
        pytest.fail("a CUDA device is required for the gpu tests")
    import paper_2609_33224_gb300 as P
    P.build()
    return P


def _same(a, b):
    for k in a:
        x, y = np.asarray(a[k]), np.asarray(b[k])
        if x.dtype == np.float32:
            assert np.array_equal(x.view(np.uint32), y.view(np.uint32)), k
        else:
            assert np.array_equal(x, y), k


@pytest.mark.parametrize("cfg", [0, 1])
def test_small_windows_match_the_whole_form_and_the_oracle(P, cfg):
    wl = W.generate(cfg)
    tw = W.tree_window(wl.window)
    assert (tw.parent >= 0).any()
    with P.scheduler_for(wl) as s:
        g_tree = s.score_window(tw, want=WANT)
        g_full = s.score_window(wl.window, want=WANT)
        d_tree = s.schedule_window(tw)
    _same(g_tree, g_full)
    orc = Oracle(wl.instances.I, wl.model).load(wl.instances)
    o = orc.score_rows(wl.window)
    for k in ("hits", "cls", "best", "path"):
        assert np.array_equal(g_tree[k], o[k]), k
    od = orc.schedule(wl.window)
    for k in ("assign", "path", "hit_chosen"):
        assert np.array_equal(d_tree[k], od[k]), k


def test_production_window_in_the_shared_prefix_form(P):
    """1024 instances x 16384 requests sent as 13.8M own blocks instead of 66.8M chain blocks."""
    with np.load(G.path("production"), allow_pickle=False) as z:
        gold = {k: z[k] for k in z.files}
    wl = W.generate(2)
    assert str(gold["input"]) == G.input_digest(wl)
    tw = W.tree_window(wl.window)
    assert int(tw.chain_off[-1]) * 4 < int(wl.window.chain_off[-1])
    R = wl.window.R
    with P.scheduler_for(wl) as s:
        g = s.score_window(tw, want=WANT)
        d = s.schedule_window(tw)
        pend = s.get_instances(pending=True)
    C = int(gold["chunk"])
    for c, a in enumerate(range(0, R, C)):
        got = G.score_digests(np.ascontiguousarray(g["hits"][a:a + C]), np.ascontiguousarray(g["tpot"][a:a + C]),
                              np.ascontiguousarray(g["ttft"][a:a + C]), np.ascontiguousarray(g["cls"][a:a + C]))
        assert got == (str(gold["hits_digest"][c]), str(gold["tpot_digest"][c]), str(gold["ttft_digest"][c]),
                       str(gold["cls_digest"][c])), c
    assert np.array_equal(g["best"], gold["best"]) and np.array_equal(g["path"], gold["score_path"])
    for k in ("assign", "path", "hit_chosen"):
        assert np.array_equal(d[k], gold[k]), k
    for k in ("qr", "q", "S"):
        assert np.array_equal(pend[k], gold["pend_" + k]), k


def test_streaming_windows_in_the_shared_prefix_form(P):
    """A reduced streaming run (64 instances, 200-request windows, 4 windows carried with commit,
    engine progress and eviction): the same decisions, state and cache sizes whichever form the
    windows are sent in."""
    over = dict(num_instances=64, window_requests=200, num_sessions=512, cap_blocks=20000)
    runs = []
    for tree in (False, True):
        wl = W.generate(4, **over)
        ins = wl.instances
        out = []
        with P.Scheduler(ins.I, ins.cap_blocks, wl.window.R, 8192 * wl.window.R, wl.model,
                         table_load_factor=wl.table_load_factor, probe_mode=P.PS_PROBE_SEARCH, track_lru=True,
                         max_active_requests=512) as s:
            s.load_workload_instances(ins)
            s.load_requests(wl.initial_requests())
            for w in range(4):
                win = wl.window if w == 0 else wl.next_window()
                g = s.schedule_window(W.tree_window(win) if tree else win)
                s.commit_window(last_use=w + 1)
                s.advance_window(20.0, 1000, evict=True)
                st = s.get_instances()
                out.append((g["assign"], g["path"], g["hit_chosen"], st["qr"], st["q"], st["S"], s.cached_blocks()))
        runs.append(out)
    for w in range(4):
        for x, y in zip(runs[0][w], runs[1][w]):
            assert np.array_equal(x, y), w


def test_malformed_links_are_refused(P):
    wl = W.generate(0)
    tw = W.tree_window(wl.window)
    with P.scheduler_for(wl) as s:
        bad = W.TreeWindow(**{k: getattr(tw, k).copy() for k in tw.__dataclass_fields__})
        r = int(np.nonzero(bad.parent >= 0)[0][0])
        bad.parent[r] = r  # not an earlier request
        with pytest.raises(P.PSError) as e:
            s.score_window(bad, want=("best",))
        assert e.value.status == P.PS_ERR_INVALID
        bad = W.TreeWindow(**{k: getattr(tw, k).copy() for k in tw.__dataclass_fields__})
        bad.parent[r] = -1  # then its own blocks must be the whole chain
        with pytest.raises(P.PSError) as e:
            s.score_window(bad, want=("best",))
        assert e.value.status == P.PS_ERR_INVALID
        # the context is still usable
        assert np.array_equal(s.score_window(tw, want=("best",))["best"],
                              s.score_window(wl.window, want=("best",))["best"])
