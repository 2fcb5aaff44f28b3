"""Failure detection of the greedy pipeline without a GPU fault: a bounded device-side wait runs out.

The pipelined greedy pass (search mode) is a cooperative launch whose thread blocks hand each other
decisions, inserted blocks and probed hit rows through flags in device memory, each wait bounded by
the context's wait limit.  Here the limit is set to 1 us on a window whose first request must cache
a 65536-block chain tail: the rows a fixed lag (21 requests) later can be probed only after that insert is done,
which takes far longer than 1 us, so some wait must give up.  The call has to return
PS_ERR_TIMEOUT (every block of the launch ended, or the call would not return), and the same context
with the default limit must then schedule the same window exactly as the oracle does.
"""
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


def _window(R, long_blocks):
    rng = np.random.default_rng(5)
    nb = np.full(R, 16, np.int64)
    nb[0] = long_blocks
    off = np.zeros(R + 1, np.uint64)
    off[1:] = np.cumsum(nb)
    hashes = rng.integers(2, 2 ** 63, int(off[-1]), dtype=np.int64).astype(np.uint64)
    return W.Window(chain_off=off, chain_hash=hashes, prompt_tokens=(16 * nb).astype(np.uint32),
                    ttft_target=np.full(R, 1e7, np.float32), tpot_target=np.full(R, 1e4, np.float32),
                    session=np.zeros(R, np.uint32), out_tokens=np.zeros(R, np.uint32))


def test_wait_limit_expires_then_the_context_recovers(P):
    I, R = 64, 40
    win = _window(R, 65536)
    ins = W.Instances(b=np.zeros(I, np.int32), qr=np.zeros(I, np.int32), q=np.zeros(I, np.int64),
                      S=np.zeros(I, np.int64), M_KV=np.full(I, 1 << 24, np.int64), B_max=np.full(I, 64, np.int32),
                      cap_blocks=np.full(I, 1 << 17, np.uint64), chain_inst=np.zeros(0, np.uint32),
                      chain_off=np.zeros(1, np.uint64), chain_hash=np.zeros(0, np.uint64),
                      chain_parent=np.zeros(0, np.uint64))
    with P.Scheduler(I, ins.cap_blocks, R, int(win.chain_off[-1]), W.MODEL_DEFAULT,
                     probe_mode=P.PS_PROBE_SEARCH) as s:
        s.load_workload_instances(ins)
        s.set_wait_limit(1000)
        with pytest.raises(P.PSError) as e:
            s.schedule_window(win)
        assert e.value.status == P.PS_ERR_TIMEOUT, str(e.value)
        with pytest.raises(P.PSError) as e2:
            s.commit_window()  # the timed-out window is not pending
        assert e2.value.status == P.PS_ERR_STATE
        s.set_wait_limit(0)
        g = s.schedule_window(win)
    o = Oracle(I, W.MODEL_DEFAULT).load(ins).schedule(win)
    for k in ("assign", "path", "hit_chosen"):
        assert np.array_equal(g[k], o[k]), k
    assert g["assign"][0] >= 0 and g["hit_chosen"][0] == 0  # the long chain was admitted cold


def test_wait_limit_bounds(P):
    with P.Scheduler(2, [16, 16], 4, 64, W.MODEL_DEFAULT) as s:
        s.set_wait_limit(5 * 10 ** 9)
        with pytest.raises(P.PSError) as e:
            s.set_wait_limit(61 * 10 ** 9)
        assert e.value.status == P.PS_ERR_INVALID
