"""Parity over whole windows at the workloads' full sizes, in the launch configuration the benchmark
times (search probe mode, device-resident inputs and outputs, the benchmark's grids).

The oracle cannot finish these windows inside a test run, so tests/golden/make_fullsize.py ran it
once over each of them and stored what it computed (only oracle/ and workload/ run there):
  * every request's independent scores against the committed state: per 256-row chunk the digest of
    the hit matrix, of the TPOT and TTFT bit patterns and of the classes, and every pick and path;
  * every greedy decision of the window in arrival order (assign, path, hit at decision) and the
    pending state they leave;
  * for the streaming workload, 50 windows carried one after another (commit, engine progress and
    leaf-first LRU eviction between them): every decision, and digests of the state and of the
    per-instance cached block counts after each window.
The GPU's outputs are compared with those element by element (digests of the same bytes for the
large score matrices: a chunk's digest matches only if every element of it is bit-identical).  A
digest of the inputs separates a generator difference from a scheduling one.

On this machine the oracle also recomputes a sample (a spread of score rows and the first greedy
decisions), which ties the stored values to the oracle as built here.  Properties that hold at any
size are checked on every decision as well.
"""
import os

import numpy as np
import pytest

import workload as W
from oracle import Oracle
from tests.golden import make_fullsize as G

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


def _golden(case):
    p = G.path(case)
    assert os.path.exists(p), f"{p} missing: run python tests/golden/make_fullsize.py {case}"
    with np.load(p, allow_pickle=False) as z:
        return {k: z[k] for k in z.files}


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


def _run_gpu(P, wl):
    """The whole window on the GPU: the scoring call with every per-pair output, then the greedy
    schedule, both on device buffers; returns host copies."""
    import torch
    win, ins = wl.window, wl.instances
    R, I = win.R, ins.I
    dwin = _device_window(win)
    with P.scheduler_for(wl, device=0, stream=torch.cuda.current_stream().cuda_stream,
                         probe_mode=P.PS_PROBE_SEARCH) as s:
        g = s.score_window(dwin, device_outputs=True)
        gd = s.schedule_window(dwin, scores=("best", "path"), device_outputs=True)
        pend = s.get_instances(pending=True)
    torch.cuda.synchronize()
    out = dict(hits=_host(g["hits"], np.uint32).reshape(R, I), tpot=_host(g["tpot"], np.float32).reshape(R, I),
               ttft=_host(g["ttft"], np.float32).reshape(R, I), cls=_host(g["cls"], np.uint8).reshape(R, I),
               best=_host(g["best"], np.int32), path=_host(g["path"], np.uint8),
               assign=_host(gd["assign"], np.int32), dpath=_host(gd["path"], np.uint8),
               hit_chosen=_host(gd["hit_chosen"], np.uint32), pend=pend)
    # the schedule call's own independent scores equal the score call's
    assert np.array_equal(_host(gd["scores"]["best"], np.int32), out["best"])
    assert np.array_equal(_host(gd["scores"]["path"], np.uint8), out["path"])
    return out


def _check_golden(case, wl, g):
    gold = _golden(case)
    assert str(gold["input"]) == G.input_digest(wl), "the generator's inputs differ from the stored ones"
    R = wl.window.R
    C = int(gold["chunk"])
    bad = []
    for c, a in enumerate(range(0, R, C)):
        got = G.score_digests(g["hits"][a:a + C], g["tpot"][a:a + C], g["ttft"][a:a + C], g["cls"][a:a + C])
        exp = (gold["hits_digest"][c], gold["tpot_digest"][c], gold["ttft_digest"][c], gold["cls_digest"][c])
        for name, x, y in zip(("hits", "tpot", "ttft", "cls"), got, exp):
            if x != str(y):
                bad.append((name, a))
    assert not bad, f"score chunks differing from the oracle's (array, first row): {bad[:8]}"
    assert np.array_equal(g["best"], gold["best"]), np.nonzero(g["best"] != gold["best"])[0][:5]
    assert np.array_equal(g["path"], gold["score_path"])
    for k, gk in (("assign", "assign"), ("dpath", "path"), ("hit_chosen", "hit_chosen")):
        assert np.array_equal(g[k], gold[gk]), (k, np.nonzero(g[k] != gold[gk])[0][:5])
    for k in ("qr", "q", "S"):
        assert np.array_equal(g["pend"][k], gold["pend_" + k]), k
    return gold


def _check_live_sample(wl, g, n_rows, n_prefix):
    """The oracle built here on a sample: score rows element by element, the greedy's first decisions."""
    win, ins = wl.window, wl.instances
    orc = Oracle(ins.I, wl.model).load(ins)
    rows = _sample_rows(win.R, n_rows)
    o = orc.score_rows(win, rows=rows)
    assert np.array_equal(g["hits"][rows], o["hits"]), np.argwhere(g["hits"][rows] != o["hits"])[:5]
    assert np.array_equal(g["cls"][rows], o["cls"])
    assert np.array_equal(g["best"][rows], o["best"]) and np.array_equal(g["path"][rows], o["path"])
    for k in ("tpot", "ttft"):
        np.testing.assert_allclose(g[k][rows], o[k], rtol=REL, atol=0)
        assert np.array_equal(g[k][rows].view(np.uint32), o[k].view(np.uint32))
    od = orc.schedule(_prefix(win, n_prefix))
    assert np.array_equal(g["assign"][:n_prefix], od["assign"])
    assert np.array_equal(g["dpath"][:n_prefix], od["path"])
    assert np.array_equal(g["hit_chosen"][:n_prefix], od["hit_chosen"])


def _check_invariants(wl, g):
    """Properties of every decision: valid picks, hits within the chain and at least the committed
    hit, rejects with hit 0, the pending state = committed state + the admitted requests."""
    win, ins = wl.window, wl.instances
    I = ins.I
    nb = np.diff(win.chain_off).astype(np.int64)
    assign, dpath, hch, hits = g["assign"], g["dpath"], g["hit_chosen"], g["hits"]
    picked = assign >= 0
    assert ((assign >= -1) & (assign < I)).all()
    assert np.array_equal(dpath == 2, ~picked)
    assert (hch[~picked] == 0).all() and (hch <= nb).all()
    rr = np.nonzero(picked)[0]
    assert (hch[rr] >= hits[rr, assign[rr]]).all()
    L = win.prompt_tokens.astype(np.int64)
    n_new = L[rr] - 16 * hch[rr].astype(np.int64)
    pend = g["pend"]
    assert np.array_equal(pend["qr"].astype(np.int64), ins.qr.astype(np.int64) + np.bincount(assign[rr], minlength=I))
    assert np.array_equal(pend["q"], ins.q + np.bincount(assign[rr], weights=n_new, minlength=I).astype(np.int64))
    assert np.array_equal(pend["S"], ins.S + np.bincount(assign[rr], weights=L[rr], minlength=I).astype(np.int64))
    assert np.array_equal(pend["b"], ins.b) and np.array_equal(pend["M_KV"], ins.M_KV)


def _whole_window(P, case, n_rows, n_prefix):
    cfg, over = G.CASES[case]
    wl = W.generate(cfg, **over)
    g = _run_gpu(P, wl)
    _check_golden(case, wl, g)
    _check_invariants(wl, g)
    _check_live_sample(wl, g, n_rows, n_prefix)
    counts = np.bincount(g["dpath"].astype(np.int64), minlength=3)
    print(f"{case}: {wl.window.R} x {wl.instances.I}, packed {counts[0]} fallback {counts[1]} reject {counts[2]}; "
          f"every score and decision equal to the oracle's")
    return counts


def test_production_window_whole(P):
    """1024 instances x 16384 requests, 200K-block caches at load factor 0.9: all 16.8M scores and
    all 16384 decisions."""
    _whole_window(P, "production", n_rows=24, n_prefix=256)


def test_production_window_packing_whole(P):
    """The production window with small queues and a 200-ms TPOT target: most independent scores
    pick from T (about 9700 of 16384), and as the window fills the instances' queues the greedy still
    packs several thousand requests by the D-C-Q key (the default window packs 47)."""
    counts = _whole_window(P, "production_packs", n_rows=16, n_prefix=128)
    assert counts[0] > 4000


def test_long_context_window_whole(P):
    """256 instances x 2048 requests, chains up to 65536 blocks, 1M-block caches: all scores and
    decisions."""
    _whole_window(P, "long_context", n_rows=16, n_prefix=64)


def test_streaming_first_50_windows(P):
    """The streaming workload at full size (1024 instances, 200K-block caches, 1000-request windows)
    for 50 windows carried one after another: every decision, and the state and per-instance cache
    sizes after each window's commit, engine progress and eviction, against the stored oracle run."""
    gold = _golden("streaming")
    wl = W.generate(4)
    assert str(gold["input"]) == G.input_digest(wl), "the generator's inputs differ from the stored ones"
    ins = wl.instances
    n = gold["assign"].shape[0]
    with P.Scheduler(ins.I, ins.cap_blocks, wl.window.R, 8192 * wl.window.R, wl.model,
                     table_load_factor=wl.table_load_factor, probe_mode=P.PS_PROBE_SEARCH, track_lru=True,
                     max_active_requests=512) as s:
        s.load_workload_instances(ins)
        s.load_requests(wl.initial_requests())
        for w in range(n):
            win = wl.window if w == 0 else wl.next_window()
            assert G.digest(win.chain_off, win.chain_hash, win.prompt_tokens, win.ttft_target, win.tpot_target,
                            win.out_tokens) == str(gold["window_digest"][w]), w
            g = s.schedule_window(win)
            for k in ("assign", "path", "hit_chosen"):
                assert np.array_equal(g[k], gold[k][w]), (w, k, np.nonzero(g[k] != gold[k][w])[0][:5])
            s.commit_window(last_use=w + 1)
            s.advance_window(20.0, 1000, evict=True)
            st = s.get_instances()
            assert G.digest(st["b"], st["qr"], st["q"], st["S"]) == str(gold["state_digest"][w]), w
            cached = s.cached_blocks()
            assert G.digest(cached.astype(np.uint64)) == str(gold["cached_digest"][w]), w
            assert (cached <= ins.cap_blocks).all()


def test_streaming_live_oracle_first_windows(P):
    """The first three streaming windows against the oracle built here: state and cache sizes each
    window, and the hits of each window's chains after eviction on sampled rows."""
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
            rows = _sample_rows(win.R, 16)
            gh = s.score_window(win, want=("hits",))["hits"][rows]
            assert np.array_equal(gh, orc.score_rows(win, rows=rows)["hits"]), w
