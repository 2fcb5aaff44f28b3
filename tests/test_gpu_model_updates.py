"""Model updates on a live context, on the GPU vs the oracle: the recompute-budget sweep through
ps_set_model (Section 8's eta study), and Section 5.3's online calibration through ps_calibrate
between streaming windows."""
import numpy as np
import pytest

import workload as W
from oracle import Oracle
from paper_2609_33224_gb300.diagnostics import PAPER_ETAS, eta_sweep

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    import torch
    if not torch.cuda.is_available():
        pytest.fail("a CUDA device is required for the gpu tests")
    import paper_2609_33224_gb300 as P
    P.build()
    return P


def _head(win, n):
    off = win.chain_off[: n + 1]
    return W.Window(chain_off=off.copy(), chain_hash=win.chain_hash[: int(off[-1])].copy(),
                    prompt_tokens=win.prompt_tokens[:n].copy(), ttft_target=win.ttft_target[:n].copy(),
                    tpot_target=win.tpot_target[:n].copy(), session=win.session[:n].copy(),
                    out_tokens=win.out_tokens[:n].copy())


@pytest.mark.parametrize("mode", [0, 1])
def test_eta_sweep_through_set_model(P, mode):
    wl = W.generate(1)
    win = _head(wl.window, 512)
    ins = wl.instances
    with P.scheduler_for(wl, probe_mode=mode, max_window_requests=win.R) as s:
        for eta in (0.0, 0.3, 1.0, 0.5):
            model = dict(wl.model, eta=eta)
            s.set_model(model)
            g = s.schedule_window(win, scores=("hits", "cls", "best", "path"))
            orc = Oracle(ins.I, model).load(ins)
            o = orc.score_rows(win)
            od = orc.schedule(win)
            for k in ("hits", "cls", "best", "path"):
                assert np.array_equal(g["scores"][k], o[k]), (eta, k)
            for k in ("assign", "path", "hit_chosen"):
                assert np.array_equal(g[k], od[k]), (eta, k)
        got = eta_sweep(s, win, wl.model, PAPER_ETAS)
    for r, eta in zip(got, PAPER_ETAS):
        orc = Oracle(ins.I, dict(wl.model, eta=eta)).load(ins)
        cls = orc.score_rows(win)["cls"]
        od = orc.schedule(win)
        el = (cls <= 2).any(axis=1)
        assert np.isclose(r["mean_C"], (cls <= 1).sum(axis=1)[el].mean())
        adm = od["path"] < 2
        assert r["cached_tokens"] == int((16 * od["hit_chosen"][adm].astype(np.int64)).sum())


def test_set_model_rejects_a_bad_model_and_keeps_the_old(P):
    wl = W.generate(0)
    with P.scheduler_for(wl) as s:
        before = s.score_window(wl.window)
        with pytest.raises(P.PSError) as e:
            s.set_model(dict(wl.model, eta=-1.0))
        assert e.value.status == P.PS_ERR_INVALID
        after = s.score_window(wl.window)
        for k in before:
            assert np.array_equal(before[k], after[k]), k


SEG_LO = [0, 16]
SLOW = [1.25, 1.6]


def test_calibration_between_streaming_windows(P):
    """After each window's progress, every decoding instance reports one forward of an engine that
    is 1.25x / 1.6x slower than the profile below / from batch 16; both sides calibrate on the same
    samples, and the next window is scheduled on the calibrated factors."""
    model = dict(W.MODEL_DEFAULT, seg_lo=SEG_LO, ema_factor=[1.0, 1.0])
    wl = W.generate(0, seed=7, cap_blocks=1 << 16)
    wl.model = model
    ins = wl.instances
    req = wl.initial_requests()
    orc = Oracle(ins.I, model, track_lru=True).load(ins)
    orc.load_requests(req)
    with P.Scheduler(ins.I, ins.cap_blocks, 64, 8192 * 64, model, table_load_factor=wl.table_load_factor,
                     probe_mode=1, track_lru=True, max_active_requests=512) as s:
        s.load_workload_instances(ins)
        s.load_requests(req)
        for w in range(6):
            win = wl.window if w == 0 else wl.next_window(24)
            win.tpot_target[:] = np.linspace(120.0, 240.0, win.R).astype(np.float32)
            g = s.schedule_window(win)
            o = orc.schedule(win, window_id=w + 1, streaming=True)
            for k in ("assign", "path", "hit_chosen"):
                assert np.array_equal(g[k], o[k]), (w, k)
            s.commit_window(last_use=w + 1)
            s.advance_window(20.0, 1000, evict=True)
            orc.advance(20.0, 1000)
            st = orc.get_state()
            live = np.nonzero(st["b"] > 0)[0]
            B = st["b"][live].astype(np.int64)
            S = st["S"][live].astype(np.int64)
            base = (8.0 + 0.15 * B) + 2e-5 * S
            t = (base * np.asarray(SLOW)[np.where(B >= 16, 1, 0)]).astype(np.float32)
            orc.calibrate(B, S, t)
            s.calibrate(B.astype(np.int32), S, t)
            assert np.array_equal(s.ema_factors()[:2].view(np.uint32), orc.ema_factors().view(np.uint32)), w
