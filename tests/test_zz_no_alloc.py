"""ps_score_window_noalloc: scoring for callers that cannot allocate device memory.

Such a caller (for example a serving process that reserves the GPU at start-up and forbids later
allocations) owns every buffer, so this test plays that caller: it lays out the cache tables itself
in the documented format, in device memory it allocated, and checks that two calls in a row give
the same hits, latencies, classes and picks as the context-based ps_score_window and as the oracle,
that a call after the first allocates nothing (the device's free memory does not move), that a
window of exactly PS_NOALLOC_MAX_PAIRS pairs over 4096 instances (the largest accepted) is scored
like the oracle scores it, and that bad table descriptors are refused before any lookup.
"""
import ctypes
import math

import numpy as np
import pytest

import workload as W
from oracle import Oracle
from tests.helpers import make_window, seq_tokens

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


def _caller_tables(ins):
    """The documented layout, built on the host: 8-slot buckets, candidate buckets
    b1 = (h * nbkt) >> 64 and b2 = (((h ^ (h >> 31)) * 0x7FB5D329728EA185) mod 2^64 * nbkt) >> 64,
    each key in the emptier candidate (b1 on ties), both-full keys in the first bucket with room after
    b1 with overflow bits on b1 and every bucket passed; about two slots per cached block."""
    I = ins.I
    M64 = (1 << 64) - 1
    per = np.bincount(ins.chain_inst, weights=np.diff(ins.chain_off).astype(np.float64), minlength=I)
    nbkt = [max(1, math.ceil(2 * int(n) / 8) + 1) for n in per]
    base = np.zeros(I, np.uint64)
    base[1:] = np.cumsum(np.array(nbkt[:-1], np.uint64) * 8)
    obase = np.zeros(I, np.uint64)
    obase[1:] = np.cumsum(np.array([(n + 63) // 64 for n in nbkt[:-1]], np.uint64))
    slots = np.zeros(int(sum(nbkt)) * 8, np.uint64)
    ovf = np.zeros(max(1, int(sum((n + 63) // 64 for n in nbkt))), np.uint64)

    def bucket(i, b):
        return slots[int(base[i]) + 8 * b: int(base[i]) + 8 * b + 8]

    def bit(i, b):
        return (int(ovf[int(obase[i]) + b // 64]) >> (b % 64)) & 1

    for c in range(ins.chain_inst.shape[0]):
        i = int(ins.chain_inst[c])
        n = nbkt[i]
        for key in ins.chain_hash[ins.chain_off[c]:ins.chain_off[c + 1]]:
            key = int(key)
            b1 = (key * n) >> 64
            b2 = ((((key ^ (key >> 31)) * 0x7FB5D329728EA185) & M64) * n) >> 64
            present = (bucket(i, b1) == key).any() or (bucket(i, b2) == key).any()
            b = b1
            while not present and bit(i, b):
                b = (b + 1) % n
                present = (bucket(i, b) == key).any()
            if present:
                continue
            e1, e2 = int((bucket(i, b1) == 0).sum()), int((bucket(i, b2) == 0).sum())
            if e1 or e2:
                tb = b1 if e1 >= e2 else b2
                line = bucket(i, tb)
                line[np.nonzero(line == 0)[0][0]] = key
                continue
            b = b1
            while True:
                w = int(obase[i]) + b // 64
                ovf[w] = np.uint64(int(ovf[w]) | (1 << (b % 64)))
                b = (b + 1) % n
                line = bucket(i, b)
                if (line == 0).any():
                    line[np.nonzero(line == 0)[0][0]] = key
                    break
    desc = np.zeros(I, dtype=np.dtype([("base", np.uint64), ("overflow_base", np.uint64),
                                       ("num_buckets", np.uint32), ("reserved", np.uint32)]))
    desc["base"], desc["overflow_base"], desc["num_buckets"] = base, obase, nbkt
    return slots, ovf, desc


def _dev(a):
    import torch
    a = np.ascontiguousarray(a)
    view = {np.dtype(np.uint64): np.int64, np.dtype(np.uint32): np.int32}.get(a.dtype)
    if a.dtype.names:
        return torch.from_numpy(a.view(np.uint8)).cuda()
    return torch.from_numpy(a.view(view) if view else a).cuda()


def _noalloc_score(P, ins, win, model, mode, tables=None, check_free=False):
    """Calls of the allocation-free entry point with caller-owned device buffers (two calls when
    check_free: the device's free memory is read around the second, after every buffer exists)."""
    import torch
    slots, ovf, desc = tables if tables is not None else _caller_tables(ins)
    d_slots, d_ovf, d_desc = _dev(slots), _dev(ovf), _dev(desc)
    st = {k: _dev(getattr(ins, k)) for k in ("b", "qr", "q", "S", "M_KV", "B_max")}
    sa = P.PsStateArrays(st["b"].data_ptr(), st["qr"].data_ptr(), st["q"].data_ptr(), st["S"].data_ptr(),
                         st["M_KV"].data_ptr(), st["B_max"].data_ptr())
    dwin = W.Window(**{k: _dev(getattr(win, k)) for k in win.__dataclass_fields__})
    pw = P.Scheduler.make_window(dwin)
    R, I = win.R, ins.I
    out = {"hits": torch.empty((R, I), dtype=torch.int32, device="cuda"),
           "tpot": torch.empty((R, I), dtype=torch.float32, device="cuda"),
           "ttft": torch.empty((R, I), dtype=torch.float32, device="cuda"),
           "cls": torch.empty((R, I), dtype=torch.uint8, device="cuda"),
           "best": torch.empty(R, dtype=torch.int32, device="cuda"),
           "path": torch.empty(R, dtype=torch.uint8, device="cuda")}
    sc = P.PsScores(*(out[k].data_ptr() for k in ("hits", "tpot", "ttft", "cls", "best", "path")), 1)
    m = P.make_model(model)

    def call():
        return P.lib().ps_score_window_noalloc(d_slots.data_ptr(), d_ovf.data_ptr(), d_desc.data_ptr(), I,
                                               ctypes.byref(sa), ctypes.byref(pw), ctypes.byref(m), int(mode),
                                               ctypes.byref(sc), torch.cuda.current_stream().cuda_stream)

    status = call()
    assert status == P.PS_OK, P.STATUS_NAMES.get(status, status)
    if check_free:
        torch.cuda.synchronize()
        free0, _ = torch.cuda.mem_get_info()
        status = call()
        torch.cuda.synchronize()
        free1, _ = torch.cuda.mem_get_info()
        assert status == P.PS_OK, P.STATUS_NAMES.get(status, status)
        assert free1 == free0, (free0, free1)
    res = {k: v.cpu().numpy() for k, v in out.items()}
    res["hits"] = res["hits"].view(np.uint32)
    return res


def _context_score(P, ins, win, model, mode):
    with P.Scheduler(ins.I, ins.cap_blocks, max(1, win.R), max(1, int(win.chain_off[-1])), model,
                     probe_mode=mode) as s:
        s.load_workload_instances(ins)
        return s.score_window(win)


def _same(a, b, rows=None):
    for k in ("hits", "cls", "best", "path"):
        got = a[k] if rows is None else a[k][rows]
        assert np.array_equal(got, b[k]), k
    for k in ("tpot", "ttft"):
        got = a[k] if rows is None else a[k][rows]
        np.testing.assert_allclose(got, b[k], rtol=REL, atol=0)


def _oracle_score(ins, win, model, rows=None):
    return Oracle(ins.I, model).load(ins).score_rows(win, rows=rows)


def _random_case(seed, I, R):
    rng = np.random.default_rng(seed)
    base = [rng.integers(0, 1 << 17, 16 * 300).astype(np.uint32) for _ in range(3)]
    reqs = []
    for _ in range(R):
        b = base[int(rng.integers(0, 3))]
        L = int(rng.integers(0, 16 * 400))
        cut = int(rng.integers(0, b.shape[0]))
        toks = b[:L] if L <= cut else np.concatenate([b[:cut], rng.integers(0, 1 << 17, L - cut).astype(np.uint32)])
        reqs.append((toks, 2000.0, float(rng.choice([20.0, 50.0]))))
    win = make_window(reqs)
    chains, inst = [], []
    for i in range(I):
        for _ in range(int(rng.integers(1, 3))):
            b = base[int(rng.integers(0, 3))]
            chains.append(W.chain_from_tokens(b[:16 * int(rng.integers(0, 300))]))
            inst.append(i)
    off = np.zeros(len(chains) + 1, np.uint64)
    off[1:] = np.cumsum([c.shape[0] for c in chains])
    ins = W.Instances(b=rng.integers(0, 40, I).astype(np.int32), qr=rng.integers(0, 5, I).astype(np.int32),
                      q=rng.integers(0, 9000, I).astype(np.int64), S=rng.integers(0, 300000, I).astype(np.int64),
                      M_KV=np.full(I, 10 ** 6, np.int64), B_max=np.full(I, 64, np.int32),
                      cap_blocks=np.full(I, 4096, np.uint64), chain_inst=np.array(inst, np.uint32), chain_off=off,
                      chain_hash=np.concatenate(chains).astype(np.uint64), chain_parent=np.zeros(len(chains), np.uint64))
    return ins, win


def test_noalloc_matches_context_scoring_on_two_calls_in_a_row(P):
    wl = W.generate(0)
    first = _noalloc_score(P, wl.instances, wl.window, wl.model, P.PS_PROBE_SEARCH)
    _same(first, _context_score(P, wl.instances, wl.window, wl.model, P.PS_PROBE_SEARCH))
    _same(first, _oracle_score(wl.instances, wl.window, wl.model))
    # the second call reuses the shared array left over from the first with other sizes
    ins, win = _random_case(11, 70, 90)
    second = _noalloc_score(P, ins, win, dict(W.MODEL_DEFAULT), P.PS_PROBE_LINEAR)
    _same(second, _context_score(P, ins, win, dict(W.MODEL_DEFAULT), P.PS_PROBE_LINEAR))
    _same(second, _oracle_score(ins, win, dict(W.MODEL_DEFAULT)))


def test_noalloc_allocates_nothing_after_set_up(P):
    """Free device memory is the same before and after a call made once every buffer exists."""
    wl = W.generate(0)
    res = _noalloc_score(P, wl.instances, wl.window, wl.model, P.PS_PROBE_SEARCH, check_free=True)
    _same(res, _oracle_score(wl.instances, wl.window, wl.model))


def _wide_case(I, R, seed=3):
    """I instances each caching a prefix of one of three token sequences (0..40 blocks) and R
    requests that share a prefix with one of them."""
    rng = np.random.default_rng(seed)
    base = [rng.integers(0, 1 << 17, 16 * 64).astype(np.uint32) for _ in range(3)]
    chains = [W.chain_from_tokens(b) for b in base]
    sel = rng.integers(0, 3, I)
    depth = rng.integers(0, 41, I)
    keep = depth > 0
    off = np.zeros(int(keep.sum()) + 1, np.uint64)
    off[1:] = np.cumsum(depth[keep])
    ins = W.Instances(b=rng.integers(0, 60, I).astype(np.int32), qr=rng.integers(0, 4, I).astype(np.int32),
                      q=rng.integers(0, 6000, I).astype(np.int64), S=rng.integers(0, 200000, I).astype(np.int64),
                      M_KV=np.full(I, 10 ** 6, np.int64), B_max=np.full(I, 128, np.int32),
                      cap_blocks=np.full(I, 64, np.uint64), chain_inst=np.nonzero(keep)[0].astype(np.uint32),
                      chain_off=off,
                      chain_hash=np.concatenate([chains[s][:d] for s, d in zip(sel[keep], depth[keep])]).astype(np.uint64),
                      chain_parent=np.zeros(int(keep.sum()), np.uint64))
    reqs = []
    for _ in range(R):
        b = base[int(rng.integers(0, 3))]
        L = int(rng.integers(16, 16 * 64))
        cut = int(rng.integers(0, L))
        toks = np.concatenate([b[:cut], rng.integers(0, 1 << 17, L - cut).astype(np.uint32)])
        reqs.append((toks, 2000.0, float(rng.choice([30.0, 60.0]))))
    return ins, make_window(reqs)


def test_noalloc_at_the_pair_limit_with_4096_instances(P):
    """R x I = PS_NOALLOC_MAX_PAIRS exactly (512 requests x 4096 instances, the largest instance
    count the call takes): sampled rows against the oracle, the window's picks against the rows."""
    I = 4096
    R = P.PS_NOALLOC_MAX_PAIRS // I
    assert R * I == P.PS_NOALLOC_MAX_PAIRS
    ins, win = _wide_case(I, R)
    res = _noalloc_score(P, ins, win, dict(W.MODEL_DEFAULT), P.PS_PROBE_SEARCH)
    rows = np.unique(np.concatenate([[0, R - 1], np.linspace(0, R - 1, 40).astype(np.int64)])).astype(np.uint32)
    _same(res, _oracle_score(ins, win, dict(W.MODEL_DEFAULT), rows=rows), rows=rows)
    assert ((res["best"] >= -1) & (res["best"] < I)).all()


def test_noalloc_rejects_bad_table_descriptors(P):
    """A descriptor whose base is not a whole bucket, one with no bucket, and a misaligned slot
    array are refused with PS_ERR_INVALID before any table is read."""
    import torch
    wl = W.generate(0)
    slots, ovf, desc = _caller_tables(wl.instances)
    for bad in ("base", "buckets"):
        d = desc.copy()
        if bad == "base":
            d["base"][3] += 1
        else:
            d["num_buckets"][5] = 0
        with pytest.raises(AssertionError, match="PS_ERR_INVALID"):
            _noalloc_score(P, wl.instances, wl.window, wl.model, P.PS_PROBE_SEARCH, tables=(slots, ovf, d))
    d_slots = _dev(np.concatenate([np.zeros(1, np.uint64), slots]))
    st = {k: _dev(getattr(wl.instances, k)) for k in ("b", "qr", "q", "S", "M_KV", "B_max")}
    sa = P.PsStateArrays(*(st[k].data_ptr() for k in ("b", "qr", "q", "S", "M_KV", "B_max")))
    dwin = W.Window(**{k: _dev(getattr(wl.window, k)) for k in wl.window.__dataclass_fields__})
    pw = P.Scheduler.make_window(dwin)
    best = torch.empty(wl.window.R, dtype=torch.int32, device="cuda")
    sc = P.PsScores(None, None, None, None, best.data_ptr(), None, 1)
    m = P.make_model(wl.model)
    status = P.lib().ps_score_window_noalloc(d_slots.data_ptr() + 8, _dev(ovf).data_ptr(), _dev(desc).data_ptr(),
                                             wl.instances.I, ctypes.byref(sa), ctypes.byref(pw), ctypes.byref(m),
                                             1, ctypes.byref(sc), torch.cuda.current_stream().cuda_stream)
    assert status == P.PS_ERR_INVALID


def test_noalloc_rejects_windows_beyond_its_fixed_scratch(P):
    import torch
    I = 1024
    R = P.PS_NOALLOC_MAX_PAIRS // I + 1
    win = make_window([(seq_tokens("A", 16), 2000.0, 50.0)] * R)
    dwin = W.Window(**{k: _dev(getattr(win, k)) for k in win.__dataclass_fields__})
    pw = P.Scheduler.make_window(dwin)
    z32 = torch.zeros(I, dtype=torch.int32, device="cuda")
    z64 = torch.zeros(I, dtype=torch.int64, device="cuda")
    sa = P.PsStateArrays(z32.data_ptr(), z32.data_ptr(), z64.data_ptr(), z64.data_ptr(), z64.data_ptr(),
                         z32.data_ptr())
    best = torch.empty(R, dtype=torch.int32, device="cuda")
    sc = P.PsScores(None, None, None, None, best.data_ptr(), None, 1)
    slots = torch.zeros(8 * I, dtype=torch.int64, device="cuda")
    ovf = torch.zeros(I, dtype=torch.int64, device="cuda")
    desc = torch.zeros(3 * I, dtype=torch.int64, device="cuda")
    m = P.make_model(dict(W.MODEL_DEFAULT))
    status = P.lib().ps_score_window_noalloc(slots.data_ptr(), ovf.data_ptr(), desc.data_ptr(), I, ctypes.byref(sa),
                                             ctypes.byref(pw), ctypes.byref(m), 1, ctypes.byref(sc),
                                             torch.cuda.current_stream().cuda_stream)
    assert status == P.PS_ERR_INVALID
