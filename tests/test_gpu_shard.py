"""Column-block scoring on the GPU: a pool's instances split over two contexts on one device, each
scoring its block (ps_shard_wmin, ps_shard_pick), merged through the library's merge layer with the
two blocks as threads of one process (shard.LocalGroup; across GPUs the same code runs over
torch.distributed).  The merged picks must equal the oracle's on the whole pool, and each block's
per-pair outputs must equal the pool's columns bit for bit (the oracle's on the small windows, the
stored oracle digests on the production window).
"""
import threading

import numpy as np
import pytest

import workload as W
from oracle import Oracle
from tests.golden import make_fullsize as G

pytestmark = pytest.mark.gpu

WANT = ("hits", "tpot", "ttft", "cls")


@pytest.fixture(scope="module")
def P():
    import torch
    if not torch.cuda.is_available():
        pytest.fail("a CUDA device is required for the gpu tests")
    import paper_2609_33224_gb300 as P
    P.build()
    return P


def _run_blocks(P, wl, cuts, model=None, device_inputs=False):
    """Score wl.window over column blocks [cuts[k], cuts[k+1]), one context and one thread each.
    Returns the merged result per block and each block's per-pair outputs (numpy)."""
    from paper_2609_33224_gb300 import shard
    import torch
    ins, win = wl.instances, wl.window
    nb = len(cuts) - 1
    grp = shard.LocalGroup(nb)
    scheds = []
    for k in range(nb):
        blk = W.column_block(ins, cuts[k], cuts[k + 1])
        s = P.Scheduler(blk.I, blk.cap_blocks, win.R, max(1, int(win.chain_off[-1])), model or wl.model,
                        table_load_factor=wl.table_load_factor, probe_mode=P.PS_PROBE_SEARCH)
        s.load_workload_instances(blk)
        scheds.append(s)
    if device_inputs:
        view = {np.dtype(np.uint64): np.int64, np.dtype(np.uint32): np.int32}
        win = W.Window(**{f: torch.from_numpy(np.ascontiguousarray(getattr(win, f)).view(
            view.get(getattr(win, f).dtype, getattr(win, f).dtype))).to("cuda:0")
            for f in win.__dataclass_fields__})
    out, errs = [None] * nb, []

    def work(k):
        try:
            torch.cuda.set_device(0)
            r = shard.score_window_sharded(scheds[k], win, cuts[k], grp.allreduce_min(k), scores=WANT,
                                           device_outputs=device_inputs)
            if device_inputs:
                r["scores"] = {n: v.cpu().numpy() for n, v in r["scores"].items()}
                r["scores"]["hits"] = r["scores"]["hits"].view(np.uint32)
            out[k] = r
        except BaseException as e:  # noqa: BLE001 - reported below
            errs.append(e)
            grp.abort()

    th = [threading.Thread(target=work, args=(k,)) for k in range(nb)]
    for t in th:
        t.start()
    for t in th:
        t.join(timeout=600)
    for s in scheds:
        s.close()
    assert not errs, errs
    return out


def _check_small(P, wl, cuts, model=None):
    m = model or wl.model
    orc = Oracle(wl.instances.I, m).load(wl.instances).score_rows(wl.window)
    out = _run_blocks(P, wl, cuts, model=m)
    for k, r in enumerate(out):
        assert np.array_equal(r["best"], orc["best"]), k
        assert np.array_equal(r["path"], orc["path"]), k
        lo, hi = cuts[k], cuts[k + 1]
        for n in WANT:
            want = orc[n][:, lo:hi]
            got = r["scores"][n]
            if n in ("tpot", "ttft"):
                assert np.array_equal(got.view(np.uint32), want.view(np.uint32)), (k, n)
            else:
                assert np.array_equal(got, want), (k, n)
    return out


@pytest.mark.parametrize("cuts", [[0, 3, 8], [0, 1, 8], [0, 2, 5, 8]])
def test_tiny_window_blocks(P, cuts):
    _check_small(P, W.generate(0), cuts)


@pytest.mark.parametrize("variant", ["eta0", "H-C-Q", "fallback_dcq", "tight"])
def test_eval_scale_window_blocks(P, variant):
    """64 instances x 4096 requests in two blocks of 24 and 40 instances, under model variants that
    move W_min's role (eta 0), the order inside T (H-C-Q with qr in the tie word), the fallback (the
    D-C-Q order over C) and the share of fallback rows (tight TPOT targets)."""
    import oracle
    wl = W.generate(1)
    m = dict(wl.model)  # the variant as both sides spell it (the oracle's keys and the library's)
    if variant == "eta0":
        m["eta"] = 0.0
    elif variant == "H-C-Q":
        m["selector"] = P.SELECTORS["H-C-Q"]
        assert oracle.SELECTORS["H-C-Q"] == m["selector"]
    elif variant == "fallback_dcq":
        m.update(P.ABLATIONS["CT"])
        m.update(oracle.ABLATIONS["CT"])
    else:
        wl.window.tpot_target[:] = np.float32(30.0)
    out = _check_small(P, wl, [0, 24, 64], model=m)
    if variant == "tight":
        assert (out[0]["path"] == 1).any() and (out[0]["path"] == 0).any()


def test_production_window_blocks(P):
    """1024 instances x 16384 requests in two blocks of 512, inputs on the device: every pick and path
    against the stored oracle run, and the blocks' columns put together against its per-chunk digests."""
    p = G.path("production")
    with np.load(p, allow_pickle=False) as z:
        gold = {k: z[k] for k in z.files}
    wl = W.generate(2)
    assert str(gold["input"]) == G.input_digest(wl)
    out = _run_blocks(P, wl, [0, 512, 1024], device_inputs=True)
    for r in out:
        assert np.array_equal(r["best"], gold["best"])
        assert np.array_equal(r["path"], gold["score_path"])
    chunk = int(gold["chunk"])
    full = {n: np.concatenate([out[0]["scores"][n], out[1]["scores"][n]], axis=1) for n in WANT}
    for c in range(wl.window.R // chunk):
        sl = slice(c * chunk, (c + 1) * chunk)
        d = G.score_digests(np.ascontiguousarray(full["hits"][sl]), np.ascontiguousarray(full["tpot"][sl]),
                            np.ascontiguousarray(full["ttft"][sl]), np.ascontiguousarray(full["cls"][sl]))
        assert d == (str(gold["hits_digest"][c]), str(gold["tpot_digest"][c]), str(gold["ttft_digest"][c]),
                     str(gold["cls_digest"][c])), c


def test_pick_needs_a_fresh_wmin_call(P):
    """ps_shard_pick refuses to run without the ps_shard_wmin of its window, and after the context
    changed since."""
    wl = W.generate(0)
    with P.scheduler_for(wl) as s:
        with pytest.raises(P.PSError) as e:
            s.shard_pick(np.zeros(wl.window.R, np.uint32), 0)
        assert e.value.status == P.PS_ERR_STATE
        w = s.shard_wmin(wl.window)
        s.score_window(wl.window, want=("best",))
        with pytest.raises(P.PSError) as e:
            s.shard_pick(w, 0)
        assert e.value.status == P.PS_ERR_STATE
        w = s.shard_wmin(wl.window)
        r = s.shard_pick(w, 0)
        full = s.score_window(wl.window, want=("best",))
        picked = r["tie"] != np.uint32(0xFFFFFFFF)
        assert np.array_equal(np.where(picked, r["tie"].astype(np.int64), -1), full["best"])
