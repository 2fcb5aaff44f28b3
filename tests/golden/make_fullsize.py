"""Writes the expected values of the full-window parity tests (tests/test_gpu_fullsize.py).

Every value here comes from the oracle (oracle/, the single-threaded restatement of Algorithm 1)
on the seeded synthetic inputs of workload/; nothing is read from the CUDA library.  The windows are
too large for the oracle to finish within a GPU test run (about 7 minutes of greedy alone for the
production window on one core), so the oracle runs here once and the test compares against what it
wrote:

  production        the production-scale window: 1024 instances x 16384 requests
  production_packs  the same window with queued prefill drawn from U{0..256}, decode batches from
                    U{0..64} and a 200-ms TPOT target, so that the packing path decides thousands of
                    requests (most independent scores pick from T)
  long_context      256 instances x 2048 requests, chains of up to 65536 blocks
  streaming         the streaming workload's first 50 windows (1024 instances, 1000 requests each),
                    with commit, engine progress and leaf-first LRU eviction between windows

For the three single windows the file holds, element by element where it is small and as digests of
256-row chunks where it is not:
  * the independent scores of every request against the committed caches and state: the blake2b
    digest of each 256-row chunk of the hit matrix, of the TPOT and TTFT bit patterns and of the
    classes; the pick and path of every request in full;
  * the greedy decisions over the whole window in arrival order (assign, path, hit at decision) and
    the pending state they leave (qr, q, S per instance).
For the stream: every window's decisions in full, and after each window's commit and progress the
digest of the state (b, qr, q, S) and of the per-instance cached block counts.
A digest of the inputs lets the test tell a generator difference from a scheduling one.

Usage: python tests/golden/make_fullsize.py [case ...]   (default: every case; about an hour with
three worker processes, each holding one oracle of 11-30 GB).
"""
from __future__ import annotations

import concurrent.futures as cf
import hashlib
import multiprocessing as mp
import os
import sys
import time

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

CHUNK = 256
STREAM_WINDOWS = 50

CASES = {
    "production": (2, {}),
    "production_packs": (2, dict(q_hi=256, b_hi=64, tpot_target_ms=200.0)),
    "long_context": (3, {}),
    "streaming": (4, {}),
}


def digest(*arrays) -> str:
    h = hashlib.blake2b(digest_size=16)
    for a in arrays:
        h.update(np.ascontiguousarray(a).tobytes())
    return h.hexdigest()


def input_digest(wl) -> str:
    win, ins = wl.window, wl.instances
    return digest(win.chain_off, win.chain_hash, win.prompt_tokens, win.ttft_target, win.tpot_target,
                  ins.b, ins.qr, ins.q, ins.S, ins.M_KV, ins.B_max, ins.chain_inst, ins.chain_off,
                  ins.chain_hash, ins.chain_parent)


def score_digests(hits, tpot, ttft, cls) -> tuple[str, str, str, str]:
    return (digest(hits), digest(tpot.view(np.uint32)), digest(ttft.view(np.uint32)), digest(cls))


def path(case: str) -> str:
    return os.path.join(HERE, f"fullsize_{case}.npz")


def _workload(case):
    import workload as W
    cfg, over = CASES[case]
    return W.generate(cfg, **over)


def job_scores(case: str, lo: int, hi: int):
    """Scores of rows [lo, hi) (a multiple of CHUNK apart): per-chunk digests, picks and paths."""
    from oracle import Oracle
    wl = _workload(case)
    orc = Oracle(wl.instances.I, wl.model).load(wl.instances)
    out = []
    for a in range(lo, hi, CHUNK):
        rows = np.arange(a, min(a + CHUNK, wl.window.R), dtype=np.uint32)
        o = orc.score_rows(wl.window, rows=rows)
        out.append((a, score_digests(o["hits"], o["tpot"], o["ttft"], o["cls"]), o["best"], o["path"]))
    return case, "scores", out


def job_greedy(case: str):
    from oracle import Oracle
    wl = _workload(case)
    orc = Oracle(wl.instances.I, wl.model).load(wl.instances)
    od = orc.schedule(wl.window)
    st = orc.get_state()
    return case, "greedy", dict(input=input_digest(wl), assign=od["assign"], path=od["path"],
                                hit_chosen=od["hit_chosen"], pend_qr=st["qr"], pend_q=st["q"], pend_S=st["S"])


def job_stream(case: str):
    from oracle import Oracle
    wl = _workload(case)
    ins = wl.instances
    inp = input_digest(wl)
    orc = Oracle(ins.I, wl.model, track_lru=True).load(ins)
    orc.load_requests(wl.initial_requests())
    A = np.zeros((STREAM_WINDOWS, wl.window.R), np.int32)
    Pth = np.zeros((STREAM_WINDOWS, wl.window.R), np.uint8)
    H = np.zeros((STREAM_WINDOWS, wl.window.R), np.uint32)
    win_d, st_d, cache_d = [], [], []
    for w in range(STREAM_WINDOWS):
        win = wl.window if w == 0 else wl.next_window()
        win_d.append(digest(win.chain_off, win.chain_hash, win.prompt_tokens, win.ttft_target, win.tpot_target,
                            win.out_tokens))
        o = orc.schedule(win, window_id=w + 1, streaming=True)
        A[w], Pth[w], H[w] = o["assign"], o["path"], o["hit_chosen"]
        orc.advance(20.0, 1000)
        st = orc.get_state()
        st_d.append(digest(st["b"], st["qr"], st["q"], st["S"]))
        cache_d.append(digest(np.array([orc.cached_blocks(i) for i in range(ins.I)], np.uint64)))
    return case, "stream", dict(input=inp, window_digest=np.array(win_d), assign=A, path=Pth, hit_chosen=H,
                                state_digest=np.array(st_d), cached_digest=np.array(cache_d))


def main(cases):
    t0 = time.time()
    jobs = []
    if "streaming" in cases:
        jobs.append((job_stream, ("streaming",)))
    for case in ("production", "production_packs", "long_context"):
        if case not in cases:
            continue
        jobs.append((job_greedy, (case,)))
        R = 16384 if CASES[case][0] == 2 else 2048
        half = (R // 2 + CHUNK - 1) // CHUNK * CHUNK
        jobs.append((job_scores, (case, 0, half)))
        jobs.append((job_scores, (case, half, R)))
    got: dict = {c: {} for c in cases}
    ctx = mp.get_context("spawn")
    with cf.ProcessPoolExecutor(max_workers=3, mp_context=ctx) as ex:
        futs = [ex.submit(f, *a) for f, a in jobs]
        for fut in cf.as_completed(futs):
            case, kind, val = fut.result()
            if kind == "scores":
                got[case].setdefault("scores", []).extend(val)
            else:
                got[case][kind] = val
            print(f"[{time.time() - t0:7.0f} s] {case} {kind} done", flush=True)
    for case in cases:
        g = got[case]
        if case == "streaming":
            np.savez_compressed(path(case), **g["stream"])
            continue
        sc = sorted(g["scores"], key=lambda x: x[0])
        d = np.array([x[1] for x in sc])
        out = dict(g["greedy"])
        out.update(chunk=np.int64(CHUNK), hits_digest=d[:, 0], tpot_digest=d[:, 1], ttft_digest=d[:, 2],
                   cls_digest=d[:, 3], best=np.concatenate([x[2] for x in sc]),
                   score_path=np.concatenate([x[3] for x in sc]))
        np.savez_compressed(path(case), **out)
        print(f"wrote {path(case)}", flush=True)


if __name__ == "__main__":
    sel = sys.argv[1:] or list(CASES)
    for c in sel:
        if c not in CASES:
            raise SystemExit(f"unknown case {c}; cases: {', '.join(CASES)}")
    main(sel)
