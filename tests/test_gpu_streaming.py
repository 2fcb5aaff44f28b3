"""Streaming windows on the GPU vs the oracle: schedule, commit, engine progress and leaf-first LRU
eviction, window after window with the state carried across windows."""
import numpy as np
import pytest

import workload as W
from oracle import Oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    import torch
    if not torch.cuda.is_available():
        pytest.fail("a CUDA device is required for the gpu tests")
    import paper_2609_33224_gb300 as P
    P.build()
    return P


def _stream(P, wl, windows, R, mode=1, max_blocks=None):
    ins = wl.instances
    req = wl.initial_requests()
    orc = Oracle(ins.I, wl.model, track_lru=True).load(ins)
    orc.load_requests(req)
    mb = max_blocks or 8192 * max(R, wl.window.R)
    with P.Scheduler(ins.I, ins.cap_blocks, max(R, wl.window.R), mb, wl.model, table_load_factor=wl.table_load_factor,
                     probe_mode=mode, track_lru=True, max_active_requests=512) as s:
        s.load_workload_instances(ins)
        s.load_requests(req)
        st_g, st_o = s.get_instances(), orc.get_state()
        for k in ("b", "qr", "q", "S"):
            assert np.array_equal(st_g[k], st_o[k]), k
        paths = []
        for w in range(windows):
            win = wl.window if w == 0 else wl.next_window(R)
            g = s.schedule_window(win)
            o = orc.schedule(win, window_id=w + 1, streaming=True)
            for k in ("assign", "path", "hit_chosen"):
                assert np.array_equal(g[k], o[k]), (w, k, np.nonzero(g[k] != o[k])[0][:5])
            paths.append(np.bincount(g["path"].astype(np.int64), minlength=3))
            s.commit_window(last_use=w + 1)
            s.advance_window(20.0, 1000, evict=True)
            orc.advance(20.0, 1000)
            st_g, st_o = s.get_instances(), orc.get_state()
            for k in ("b", "qr", "q", "S"):
                assert np.array_equal(st_g[k], st_o[k]), (w, k)
            cached = s.cached_blocks()
            assert [int(x) for x in cached] == [orc.cached_blocks(i) for i in range(ins.I)], w
            # cache contents: hit lengths of this window's chains on every instance
            assert np.array_equal(s.score_window(win, want=("hits",))["hits"], orc.score_rows(win)["hits"]), w
        return np.array(paths)


@pytest.mark.parametrize("mode", [0, 1])
def test_stream_small_with_eviction(P, mode):
    """8 instances, capacity 3000 blocks, 10 windows of 24 requests: every window evicts."""
    wl = W.generate(0, seed=5, cap_blocks=3000, fill_lo=0.8, fill_hi=1.0)
    paths = _stream(P, wl, windows=10, R=24, mode=mode)
    assert paths[:, :2].sum() > 0


def test_stream_config4_shape_reduced(P):
    """The streaming configuration's rules and mix on 64 instances, 12 windows of 200 requests."""
    wl = W.generate(4, num_instances=64, window_requests=200, num_sessions=512, cap_blocks=20000)
    paths = _stream(P, wl, windows=12, R=200)
    print("packed/fallback/reject per window:", paths.tolist())
    assert paths[:, :2].sum() > 0


def test_advance_requires_commit_and_tracking(P):
    wl = W.generate(0)
    ins = wl.instances
    with P.Scheduler(ins.I, ins.cap_blocks, 64, 65536, wl.model, track_lru=True, max_active_requests=64) as s:
        s.load_workload_instances(ins)
        s.schedule_window(wl.window)
        with pytest.raises(P.PSError) as e:
            s.advance_window()
        assert e.value.status == P.PS_ERR_STATE
        s.commit_window(1)
        s.advance_window()
    with P.Scheduler(ins.I, ins.cap_blocks, 64, 65536, wl.model) as s:
        with pytest.raises(P.PSError) as e:
            s.advance_window()
        assert e.value.status == P.PS_ERR_STATE
