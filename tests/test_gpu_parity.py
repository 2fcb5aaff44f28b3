"""CUDA path vs the oracle, element by element, through the C ABI.

Hit lengths, admission classes, picks and greedy assignments must match exactly; predicted
latencies must match within 1e-5 relative (both sides evaluate the same fp32 operations in the
same order, so they are in fact compared bit for bit as well).
"""
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


def _oracle(model, ins):
    return Oracle(ins.I, model).load(ins)


MODES = [0, 1]  # PS_PROBE_LINEAR, PS_PROBE_SEARCH


def _sched(P, model, ins, win, max_blocks=None, mode=1):
    s = P.Scheduler(ins.I, ins.cap_blocks, max(1, win.R), max(1, max_blocks or int(win.chain_off[-1])),
                    model, table_load_factor=0.5, probe_mode=mode)
    s.load_workload_instances(ins)
    return s


def _assert_scores(g, o, exact_floats=True):
    assert np.array_equal(g["hits"], o["hits"]), np.argwhere(g["hits"] != o["hits"])[:5]
    assert np.array_equal(g["cls"], o["cls"]), np.argwhere(g["cls"] != o["cls"])[:5]
    assert np.array_equal(g["best"], o["best"])
    assert np.array_equal(g["path"], o["path"])
    for k in ("tpot", "ttft"):
        np.testing.assert_allclose(g[k], o[k], rtol=REL, atol=0)
        if exact_floats:
            assert np.array_equal(g[k].view(np.uint32), o[k].view(np.uint32)), k


def _check_window(P, model, ins, win, commit=True, mode=1):
    """Score and schedule one window on both sides and compare everything."""
    orc = _oracle(model, ins)
    with _sched(P, model, ins, win, mode=mode) as s:
        g = s.score_window(win)
        o = orc.score_rows(win)
        _assert_scores(g, o)
        gd = s.schedule_window(win, scores=("hits", "best", "path"))
        od = orc.schedule(win)
        assert np.array_equal(gd["scores"]["hits"], o["hits"])
        assert np.array_equal(gd["scores"]["best"], o["best"])
        assert np.array_equal(gd["assign"], od["assign"]), np.nonzero(gd["assign"] != od["assign"])[0][:5]
        assert np.array_equal(gd["path"], od["path"])
        assert np.array_equal(gd["hit_chosen"], od["hit_chosen"])
        pend = s.get_instances(pending=True)
        ost = orc.get_state()
        for k in ("b", "qr", "q", "S", "M_KV", "B_max"):
            assert np.array_equal(pend[k], ost[k]), k
        committed = s.get_instances()
        assert np.array_equal(committed["q"], ins.q)  # pending until commit
        if commit:
            s.commit_window(last_use=1)
            after = s.get_instances()
            for k in ("qr", "q", "S"):
                assert np.array_equal(after[k], ost[k]), k
            cached = s.cached_blocks()
            for i in range(ins.I):
                assert int(cached[i]) == orc.cached_blocks(i), i
            # the committed caches now give the greedy's end-of-window hits
            g2 = s.score_window(win, want=("hits",))
            o2 = orc.score_rows(win)
            assert np.array_equal(g2["hits"], o2["hits"])
        return gd, od


@pytest.mark.parametrize("mode", MODES)
def test_hand_example_through_the_abi(P, hand, mode):
    model, ins, win, d = hand
    with _sched(P, model, ins, win, mode=mode) as s:
        g = s.score_window(win)
        e = d["score_mode"]
        assert g["hits"].tolist() == e["hits"]
        assert g["cls"].tolist() == e["cls"]
        assert g["best"].tolist() == e["best"] and g["path"].tolist() == e["path"]
        gd = s.schedule_window(win)
        e = d["schedule_mode"]
        assert gd["assign"].tolist() == e["assign"]
        assert gd["path"].tolist() == e["path"]
        assert gd["hit_chosen"].tolist() == e["hit_chosen"]
        pend = s.get_instances(pending=True)
        for i, f in enumerate(e["final_state"]):
            for k in ("b", "qr", "q", "S"):
                assert int(pend[k][i]) == f[k]
    _check_window(P, model, ins, win, mode=mode)


@pytest.mark.parametrize("mode", MODES)
def test_config0_full_parity(P, mode):
    wl = W.generate(0)
    gd, od = _check_window(P, wl.model, wl.instances, wl.window, mode=mode)
    assert (od["path"] == 0).any()


@pytest.mark.parametrize("variant", ["paper_form", "no_ttft", "ema", "eta0", "tight", "flat"])
def test_config0_model_variants(P, variant):
    wl = W.generate(0)
    m = dict(wl.model)
    win = wl.window
    if variant == "paper_form":
        m["interference_mode"] = 1
    elif variant == "no_ttft":
        m["ttft_filter"] = 0
    elif variant == "ema":
        m.update(seg_lo=[0, 9, 17, 33, 49], ema_factor=[1.0, 1.1, 1.35, 1.7, 2.0])
    elif variant == "eta0":
        m["eta"] = 0.0
    elif variant == "tight":
        win = W.Window(**{k: getattr(win, k) for k in win.__dataclass_fields__})
        win.tpot_target = np.full(win.R, 20.0, np.float32)
        win.ttft_target = np.full(win.R, 30.0, np.float32)
    elif variant == "flat":
        m.update(a1=0.0, a2=0.0, a3=0.0)  # Z = 0: every capacity-eligible instance stays in C
    _check_window(P, m, wl.instances, win)


def _random_case(seed, I, R):
    """Ragged random window: shared-prefix token trees, chains of 0..600 blocks, mixed state."""
    rng = np.random.default_rng(seed)
    base = [rng.integers(0, 1 << 17, 16 * 700).astype(np.uint32) for _ in range(4)]
    reqs = []
    for _ in range(R):
        b = base[int(rng.integers(0, 4))]
        cut = int(rng.integers(0, b.shape[0]))
        L = int(rng.integers(0, 16 * 600))
        if L <= cut:
            toks = b[:L]
        else:
            toks = np.concatenate([b[:cut], rng.integers(0, 1 << 17, L - cut).astype(np.uint32)])
        reqs.append((toks, float(rng.choice([500.0, 2000.0])), float(rng.choice([15.0, 30.0, 50.0]))))
    win = make_window(reqs)
    chains, inst = [], []
    for i in range(I):
        for _ in range(int(rng.integers(0, 4))):
            b = base[int(rng.integers(0, 4))]
            n = int(rng.integers(0, b.shape[0] // 16))
            chains.append(W.chain_from_tokens(b[:16 * n]))
            inst.append(i)
    off = np.zeros(len(chains) + 1, np.uint64)
    off[1:] = np.cumsum([c.shape[0] for c in chains]) if chains else []
    bmax = rng.integers(1, 80, I).astype(np.int32)
    ins = W.Instances(
        b=rng.integers(0, 40, I).astype(np.int32), qr=rng.integers(0, 6, I).astype(np.int32),
        q=rng.integers(0, 20000, I).astype(np.int64), S=rng.integers(0, 400000, I).astype(np.int64),
        M_KV=rng.integers(100000, 800000, I).astype(np.int64), B_max=bmax,
        cap_blocks=np.full(I, 4096, np.uint64), chain_inst=np.array(inst, np.uint32), chain_off=off,
        chain_hash=(np.concatenate(chains).astype(np.uint64) if chains else np.zeros(0, np.uint64)),
        chain_parent=np.zeros(len(chains), np.uint64))
    return ins, win


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("seed,I,R", [(1, 1, 7), (2, 3, 64), (3, 33, 37), (4, 70, 200), (5, 130, 150),
                                      (6, 8, 1), (7, 257, 90), (8, 1100, 40)])
def test_random_ragged_windows(P, seed, I, R, mode):
    ins, win = _random_case(seed, I, R)
    _check_window(P, dict(W.MODEL_DEFAULT), ins, win, mode=mode)


def test_linear_mode_is_exact_on_a_cache_that_is_not_prefix_closed(P):
    """A gapped cache (blocks 0-2 and 5-29 of a chain): linear walks stop at block 3, like the
    oracle; search mode refuses to build such a cache."""
    ch = W.chain_from_tokens(seq_tokens("A", 16 * 40))
    model = dict(W.MODEL_DEFAULT)
    win = make_window([(seq_tokens("A", 16 * 40), 2000.0, 50.0), (seq_tokens("A", 16 * 4), 2000.0, 50.0)])
    orc = Oracle(2, model)
    orc.insert_chain(0, ch[:3])
    orc.insert_chain(0, ch[5:30], parent=int(ch[4]))
    st = dict(b=np.array([3, 1], np.int32), qr=np.zeros(2, np.int32), q=np.zeros(2, np.int64),
              S=np.zeros(2, np.int64), M_KV=np.full(2, 10 ** 7, np.int64), B_max=np.full(2, 64, np.int32))
    orc.set_state(**st)
    with P.Scheduler(2, [4096, 4096], 2, 64, model, probe_mode=0) as s:
        s.insert_blocks(0, ch[:3])
        s.insert_blocks(0, ch[5:30], parent=int(ch[4]))
        s.load_instances(**st)
        g = s.score_window(win)
        o = orc.score_rows(win)
        _assert_scores(g, o)
        assert g["hits"][0].tolist() == [3, 0]
        gd, od = s.schedule_window(win), orc.schedule(win)
        assert np.array_equal(gd["assign"], od["assign"]) and np.array_equal(gd["hit_chosen"], od["hit_chosen"])
    with P.Scheduler(2, [4096, 4096], 2, 64, model, probe_mode=1) as s:
        s.insert_blocks(0, ch[:3])
        with pytest.raises(P.PSError) as e:
            s.insert_blocks(0, ch[5:30], parent=int(ch[4]))
        assert e.value.status == P.PS_ERR_INVALID


def test_empty_window_and_short_prompts(P):
    wl = W.generate(0)
    ins = wl.instances
    empty = make_window([])
    with _sched(P, wl.model, ins, empty, max_blocks=16) as s:
        g = s.score_window(empty)
        assert g["best"].shape == (0,)
        gd = s.schedule_window(empty)
        assert gd["assign"].shape == (0,)
    short = make_window([(seq_tokens("A", L), 2000.0, 50.0) for L in (0, 1, 15, 16, 17)])
    _check_window(P, wl.model, ins, short)


def test_device_inputs_and_outputs_match_host(P):
    import torch
    wl = W.generate(0)
    win = wl.window
    dwin = W.Window(**{k: torch.from_numpy(np.ascontiguousarray(getattr(win, k)).view(
        np.int64 if getattr(win, k).dtype == np.uint64 else (np.int32 if getattr(win, k).dtype == np.uint32
                                                              else getattr(win, k).dtype))).cuda()
        for k in win.__dataclass_fields__})
    with _sched(P, wl.model, wl.instances, win) as s:
        host = s.score_window(win)
        dev = s.score_window(dwin, device_outputs=True)
        for k in host:
            got = dev[k].cpu().numpy()
            assert np.array_equal(got.view(host[k].dtype) if got.dtype != host[k].dtype else got, host[k]), k
        hd = s.schedule_window(win)
        dd = s.schedule_window(dwin, device_outputs=True)
        assert np.array_equal(dd["assign"].cpu().numpy(), hd["assign"])
        assert np.array_equal(dd["hit_chosen"].cpu().numpy().view(np.uint32), hd["hit_chosen"])


def test_invalid_windows_are_rejected(P):
    wl = W.generate(0)
    win = wl.window
    with _sched(P, wl.model, wl.instances, win) as s:
        bad = W.Window(**{k: getattr(win, k).copy() for k in win.__dataclass_fields__})
        bad.prompt_tokens[3] += 16  # chain length no longer L/16
        with pytest.raises(P.PSError) as e:
            s.score_window(bad)
        assert e.value.status == P.PS_ERR_INVALID
        with pytest.raises(P.PSError) as e:
            s.commit_window()
        assert e.value.status == P.PS_ERR_STATE
        with pytest.raises(P.PSError) as e:
            s.insert_blocks(0, np.array([5, 0, 7], np.uint64))
        assert e.value.status == P.PS_ERR_INVALID
        # the context still works after errors
        g = s.score_window(win, want=("best",))
        assert g["best"].shape == (win.R,)


def test_capacity_and_table_full_errors(P):
    model = dict(W.MODEL_DEFAULT)
    # capacity 20 at load factor 0.9: ceil(20 / 0.9) = 23 slots -> 3 buckets of 8 = 24 slots
    with P.Scheduler(2, [20, 20], 4, 64, model, table_load_factor=0.9) as s:
        ch = np.arange(1, 40, dtype=np.uint64) * np.uint64(0x9E3779B97F4A7C15) % np.uint64(1 << 63) + np.uint64(1)
        with pytest.raises(P.PSError) as e:
            s.insert_blocks(0, ch[:22])
        assert e.value.status == P.PS_ERR_CAPACITY
        assert int(s.cached_blocks()[0]) == 22
        with pytest.raises(P.PSError) as e:
            s.insert_blocks(0, ch[22:30], parent=int(ch[21]))
        assert e.value.status == P.PS_ERR_TABLE_FULL
        assert int(s.cached_blocks()[0]) == 24


@pytest.mark.parametrize("mode", MODES)
def test_overflow_runs_at_high_load_factor(P, mode):
    """Tables at 95% load: many keys find both candidate buckets full and go to the overflow run;
    hits must still equal the oracle's."""
    rng = np.random.default_rng(21)
    I, cap = 3, 2000
    bases = [rng.integers(0, 1 << 17, 16 * 900).astype(np.uint32) for _ in range(3)]
    chains, inst = [], []
    for i in range(I):
        n_seq = W.chain_from_tokens(bases[i][:16 * 800])
        chains.append(n_seq)
        inst.append(i)
        filler = (rng.integers(1, 1 << 62, cap - 800, dtype=np.int64)).astype(np.uint64)
        chains.append(filler)
        inst.append(i)
    off = np.zeros(len(chains) + 1, np.uint64)
    off[1:] = np.cumsum([c.shape[0] for c in chains])
    ins = W.Instances(b=np.array([5, 9, 1], np.int32), qr=np.zeros(I, np.int32), q=np.zeros(I, np.int64),
                      S=np.zeros(I, np.int64), M_KV=np.full(I, 10 ** 8, np.int64), B_max=np.full(I, 64, np.int32),
                      cap_blocks=np.full(I, cap, np.uint64), chain_inst=np.array(inst, np.uint32), chain_off=off,
                      chain_hash=np.concatenate(chains).astype(np.uint64), chain_parent=np.zeros(len(chains), np.uint64))
    reqs = [(bases[int(rng.integers(0, 3))][:int(rng.integers(0, 16 * 900))], 2000.0, 50.0) for _ in range(60)]
    win = make_window(reqs)
    model = dict(W.MODEL_DEFAULT)
    orc = _oracle(model, ins)
    with P.Scheduler(I, ins.cap_blocks, win.R, int(win.chain_off[-1]), model, table_load_factor=0.95,
                     probe_mode=mode) as s:
        s.load_workload_instances(ins)
        assert s.cached_blocks().tolist() == [cap] * I
        g = s.score_window(win)
        _assert_scores(g, orc.score_rows(win))
        gd, od = s.schedule_window(win), orc.schedule(win)
        assert np.array_equal(gd["assign"], od["assign"]) and np.array_equal(gd["hit_chosen"], od["hit_chosen"])


@pytest.mark.parametrize("tpot,mode", [(30.0, 1), (50.0, 1), (50.0, 0)])
def test_config1_full_parity(P, tpot, mode):
    wl = W.generate(1, tpot_target_ms=tpot)
    gd, od = _check_window(P, wl.model, wl.instances, wl.window, commit=(tpot == 50.0), mode=mode)
    counts = np.bincount(od["path"], minlength=3)
    print(f"config 1 tpot {tpot}: packed {counts[0]} fallback {counts[1]} reject {counts[2]}")


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("seed,I,R", [(9, 2048, 48), (10, 1537, 33), (11, 2047, 5)])
def test_random_ragged_windows_at_the_instance_limit(P, seed, I, R, mode):
    """The largest context ps_create accepts (2048 instances; probe and summary threads then hold 8
    instances each), and ragged counts just below it."""
    ins, win = _random_case(seed, I, R)
    _check_window(P, dict(W.MODEL_DEFAULT), ins, win, mode=mode)


def test_instance_limit_is_enforced(P):
    with pytest.raises(P.PSError):
        P.Scheduler(2049, np.full(2049, 64, np.uint64), 4, 64, dict(W.MODEL_DEFAULT))
