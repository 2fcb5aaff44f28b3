"""Parity at the workloads' full sizes, in the launch configuration the benchmark times.

The GPU scores and schedules the whole window with device-resident inputs and outputs (search
probe mode, the benchmark's grid).  The oracle cannot finish these windows in seconds, so it checks
samples it can compute one by one:
  * scoring rows are independent, so a spread of rows (first, last and evenly spaced ones) is
    compared element by element (hits, classes, picks bit-exact; latencies within 1e-5 relative,
    in fact bit for bit);
  * a greedy decision depends on every earlier decision of the window, so the oracle runs the greedy
    over a prefix of the window and the GPU's decisions on that prefix must match exactly;
  * for the rest of the window, properties that hold at any size: every pick is a valid instance,
    its hit is within the chain and at least the hit against the committed caches, rejects carry
    hit 0, and the pending state equals the committed state plus the admitted requests.
"""
import numpy as np
import pytest

import workload as W
from oracle import Oracle

pytestmark = pytest.mark.gpu

REL = 1e-5


@pytest.fixture(scope="module")
def P():
    import torch
    if not torch.cuda.is_available():
        pytest.fail("a CUDA device is required for the gpu tests")
    import paper_2609_33224_gb300 as P
    P.build()
    return P


def _device_window(win):
    import torch
    view = {np.dtype(np.uint64): np.int64, np.dtype(np.uint32): np.int32}

    def dev(a):
        a = np.ascontiguousarray(a)
        return torch.from_numpy(a.view(view.get(a.dtype, a.dtype))).to("cuda:0")

    return W.Window(**{k: dev(getattr(win, k)) for k in win.__dataclass_fields__})


def _host(t, dtype):
    return t.cpu().numpy().view(dtype)


def _prefix(win, n):
    return W.Window(chain_off=win.chain_off[:n + 1].copy(), chain_hash=win.chain_hash[:int(win.chain_off[n])],
                    prompt_tokens=win.prompt_tokens[:n], ttft_target=win.ttft_target[:n],
                    tpot_target=win.tpot_target[:n], session=win.session[:n], out_tokens=win.out_tokens[:n])


def _sample_rows(R, n):
    return np.unique(np.concatenate([[0, 1, R - 1], np.linspace(0, R - 1, n).astype(np.int64)])).astype(np.uint32)


def _check_full(P, wl, n_rows, n_prefix):
    import torch
    win, ins = wl.window, wl.instances
    R, I = win.R, ins.I
    nb = np.diff(win.chain_off).astype(np.int64)
    dwin = _device_window(win)
    with P.scheduler_for(wl, device=0, stream=torch.cuda.current_stream().cuda_stream,
                         probe_mode=P.PS_PROBE_SEARCH) as s:
        g = s.score_window(dwin, device_outputs=True)
        gd = s.schedule_window(dwin, scores=("best", "path"), device_outputs=True)
        pend = s.get_instances(pending=True)
    torch.cuda.synchronize()
    hits = _host(g["hits"], np.uint32).reshape(R, I)
    tpot = _host(g["tpot"], np.float32).reshape(R, I)
    ttft = _host(g["ttft"], np.float32).reshape(R, I)
    cls = _host(g["cls"], np.uint8).reshape(R, I)
    best = _host(g["best"], np.int32)
    path = _host(g["path"], np.uint8)
    assign = _host(gd["assign"], np.int32)
    dpath = _host(gd["path"], np.uint8)
    hch = _host(gd["hit_chosen"], np.uint32)
    # the schedule call's own independent scores equal the score call's
    assert np.array_equal(_host(gd["scores"]["best"], np.int32), best)
    assert np.array_equal(_host(gd["scores"]["path"], np.uint8), path)

    orc = Oracle(I, wl.model).load(ins)
    rows = _sample_rows(R, n_rows)
    o = orc.score_rows(win, rows=rows)
    assert np.array_equal(hits[rows], o["hits"]), np.argwhere(hits[rows] != o["hits"])[:5]
    assert np.array_equal(cls[rows], o["cls"])
    assert np.array_equal(best[rows], o["best"]) and np.array_equal(path[rows], o["path"])
    for got, exp in ((tpot[rows], o["tpot"]), (ttft[rows], o["ttft"])):
        np.testing.assert_allclose(got, exp, rtol=REL, atol=0)
        assert np.array_equal(got.view(np.uint32), exp.view(np.uint32))

    od = orc.schedule(_prefix(win, n_prefix))
    assert np.array_equal(assign[:n_prefix], od["assign"]), np.nonzero(assign[:n_prefix] != od["assign"])[0][:5]
    assert np.array_equal(dpath[:n_prefix], od["path"])
    assert np.array_equal(hch[:n_prefix], od["hit_chosen"])

    # whole window: properties of every decision
    picked = assign >= 0
    assert ((assign >= -1) & (assign < I)).all()
    assert np.array_equal(dpath == 2, ~picked)
    assert (hch[~picked] == 0).all()
    assert (hch <= nb).all()
    rr = np.nonzero(picked)[0]
    assert (hch[rr] >= hits[rr, assign[rr]]).all()  # the window's own inserts only add blocks
    L = win.prompt_tokens.astype(np.int64)
    n_new = L[rr] - 16 * hch[rr].astype(np.int64)
    exp_qr = ins.qr.astype(np.int64) + np.bincount(assign[rr], minlength=I)
    exp_q = ins.q + np.bincount(assign[rr], weights=n_new, minlength=I).astype(np.int64)
    exp_S = ins.S + np.bincount(assign[rr], weights=L[rr], minlength=I).astype(np.int64)
    assert np.array_equal(pend["qr"].astype(np.int64), exp_qr)
    assert np.array_equal(pend["q"], exp_q) and np.array_equal(pend["S"], exp_S)
    assert np.array_equal(pend["b"], ins.b) and np.array_equal(pend["M_KV"], ins.M_KV)
    counts = np.bincount(dpath.astype(np.int64), minlength=3)
    print(f"{R} x {I}: packed {counts[0]} fallback {counts[1]} reject {counts[2]}; "
          f"{rows.shape[0]} rows and the first {n_prefix} decisions checked against the oracle")
    return counts


def test_production_window_full_size(P):
    """1024 instances x 16384 requests, 200K-block caches at load factor 0.9."""
    _check_full(P, W.generate(2), n_rows=48, n_prefix=768)


def test_long_context_window_full_size(P):
    """256 instances x 2048 requests, chains up to 65536 blocks, 1M-block caches."""
    _check_full(P, W.generate(3), n_rows=24, n_prefix=96)


def test_streaming_full_size_first_windows(P):
    """The streaming workload at full size (1024 instances, 200K-block caches, 1000-request windows):
    the first three windows with commit, engine progress and leaf-first LRU eviction, state and
    cache sizes compared after each window; hits of each window's chains after eviction compared on
    sampled rows."""
    wl = W.generate(4)
    ins = wl.instances
    req = wl.initial_requests()
    orc = Oracle(ins.I, wl.model, track_lru=True).load(ins)
    orc.load_requests(req)
    with P.Scheduler(ins.I, ins.cap_blocks, wl.window.R, 8192 * wl.window.R, wl.model,
                     table_load_factor=wl.table_load_factor, probe_mode=P.PS_PROBE_SEARCH, track_lru=True,
                     max_active_requests=512) as s:
        s.load_workload_instances(ins)
        s.load_requests(req)
        for w in range(3):
            win = wl.window if w == 0 else wl.next_window()
            g = s.schedule_window(win)
            o = orc.schedule(win, window_id=w + 1, streaming=True)
            for k in ("assign", "path", "hit_chosen"):
                assert np.array_equal(g[k], o[k]), (w, k, np.nonzero(g[k] != o[k])[0][:5])
            s.commit_window(last_use=w + 1)
            s.advance_window(20.0, 1000, evict=True)
            orc.advance(20.0, 1000)
            st_g, st_o = s.get_instances(), orc.get_state()
            for k in ("b", "qr", "q", "S"):
                assert np.array_equal(st_g[k], st_o[k]), (w, k)
            cached = s.cached_blocks()
            assert [int(x) for x in cached] == [orc.cached_blocks(i) for i in range(ins.I)], w
            assert (cached <= ins.cap_blocks).all()
            rows = _sample_rows(win.R, 16)
            gh = s.score_window(win, want=("hits",))["hits"][rows]
            assert np.array_equal(gh, orc.score_rows(win, rows=rows)["hits"]), w
