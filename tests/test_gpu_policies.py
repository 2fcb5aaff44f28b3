"""Policy variants of the evaluation on the CUDA path, against the oracle, through the C ABI.

Table 3's admission ablations (G: no KVC-first filter and no SLO admission, C: the filter only, T:
the SLO admission only, CT: both, each with the D-C-Q fallback) and Table 4's instance orders inside
T (D, D-Q, D-C, D-Q-C, H-C-Q; D-C-Q is the default every other test runs).  Each variant is set on
both sides (the oracle's own model keys and the library's ps_model switches, which share nothing)
and compared element by element: hits, classes, picks and every greedy decision exactly, latencies
bit for bit.  The hand-worked request of the oracle's policy pins (eight instances, one request)
runs first, so each variant's pick there is the one that test derives by hand.
"""
import numpy as np
import pytest

import oracle
import workload as W
from oracle import Oracle
from tests.helpers import make_window, seq_tokens
from tests.test_gpu_parity import _check_window

pytestmark = pytest.mark.gpu

VARIANTS = ["G", "C", "T", "CT", "D", "D-Q", "D-C", "D-Q-C", "H-C-Q"]


@pytest.fixture(scope="module")
def P():
    import torch
    if not torch.cuda.is_available():
        pytest.fail("a CUDA device is required for the gpu tests")
    import paper_2609_33224_gb300 as P
    P.build()
    return P


def _model(P, base, name):
    """The variant as both sides spell it: the oracle's keys and the library's keys in one dict."""
    m = dict(base)
    if name in oracle.ABLATIONS:
        m.update(oracle.ABLATIONS[name])
        m.update(P.ABLATIONS[name])
    else:
        m["selector"] = oracle.SELECTORS[name]
        assert P.SELECTORS[name] == m["selector"]
    return m


# The oracle policy pins' request (tests/test_oracle_policies.py header): expected picks per variant
# at a 50-ms TPOT target, and per ablation at a 5-ms target where T is empty.
TOKENS = seq_tokens("A", 1600)
STATE = dict(b=[10, 12, 12, 12, 12, 12, 20, 40], qr=[2, 3, 3, 1, 2, 1, 0, 0],
             q=[2000, 0, 0, 0, 0, 0, 0, 20000], hit=[90, 45, 60, 45, 60, 50, 0, 90])


def _hand_instances():
    chain = W.chain_from_tokens(TOKENS)
    chains = [chain[:h] for h in STATE["hit"] if h]
    inst = [i for i, h in enumerate(STATE["hit"]) if h]
    off = np.zeros(len(chains) + 1, np.uint64)
    off[1:] = np.cumsum([c.shape[0] for c in chains])
    return W.Instances(b=np.array(STATE["b"], np.int32), qr=np.array(STATE["qr"], np.int32),
                       q=np.array(STATE["q"], np.int64), S=np.zeros(8, np.int64), M_KV=np.full(8, 10 ** 9, np.int64),
                       B_max=np.full(8, 1000, np.int32), cap_blocks=np.full(8, 4096, np.uint64),
                       chain_inst=np.array(inst, np.uint32), chain_off=off,
                       chain_hash=np.concatenate(chains).astype(np.uint64), chain_parent=np.zeros(len(chains), np.uint64))


@pytest.mark.parametrize("name", VARIANTS)
@pytest.mark.parametrize("tpot", [50.0, 5.0])
def test_hand_request_every_variant(P, name, tpot):
    ins = _hand_instances()
    win = make_window([(TOKENS, 1e6, tpot)])
    m = _model(P, W.MODEL_DEFAULT, name)
    o = Oracle(8, m).load(ins).score_rows(win)
    with P.Scheduler(8, ins.cap_blocks, 1, 128, m, probe_mode=P.PS_PROBE_SEARCH) as s:
        s.load_workload_instances(ins)
        g = s.score_window(win)
        gd = s.schedule_window(win)
    for k in ("hits", "cls", "best", "path"):
        assert np.array_equal(g[k], o[k]), (name, k, g[k], o[k])
    assert gd["assign"][0] == o["best"][0] and gd["path"][0] == o["path"][0]


@pytest.mark.parametrize("name", VARIANTS)
@pytest.mark.parametrize("mode", [0, 1])
def test_config0_every_variant(P, name, mode):
    wl = W.generate(0)
    _check_window(P, _model(P, wl.model, name), wl.instances, wl.window, mode=mode)


@pytest.mark.parametrize("name", VARIANTS)
def test_config1_every_variant(P, name):
    """64 instances x 4096 requests: the variants change which path most requests take (G and C
    admit every pair of C into T, so every request packs)."""
    wl = W.generate(1)
    gd, od = _check_window(P, _model(P, wl.model, name), wl.instances, wl.window, commit=False)
    counts = np.bincount(od["path"], minlength=3)
    if name in ("G", "C"):
        assert counts[0] == (od["path"] != 2).sum()
