"""The shared-prefix (prefix-tree) form of a window: workload.tree_window keeps each request's own
blocks and a parent link to an earlier request whose whole chain starts its own.  Rebuilding every
chain from the links (root first, each ancestor's own blocks in place) must give back the window's
chains exactly, and every link must point to an earlier request whose chain is a prefix."""
import numpy as np
import pytest

import workload as W


def _rebuild(tw):
    own = tw.chain_off.astype(np.int64)
    chains = []
    for r in range(tw.R):
        p = int(tw.parent[r])
        base = chains[p] if p >= 0 else np.zeros(0, np.uint64)
        chains.append(np.concatenate([base, tw.chain_hash[own[r]:own[r + 1]]]))
    return chains


@pytest.mark.parametrize("cfg", [0, 1])
def test_round_trip_and_links(cfg):
    win = W.generate(cfg).window
    tw = W.tree_window(win)
    off = win.chain_off.astype(np.int64)
    chains = _rebuild(tw)
    for r in range(win.R):
        assert np.array_equal(chains[r], win.chain_hash[off[r]:off[r + 1]]), r
        p = int(tw.parent[r])
        if p >= 0:
            assert p < r and tw.session[p] == tw.session[r]
            n = int(off[p + 1] - off[p])
            assert np.array_equal(win.chain_hash[off[r]:off[r] + n], win.chain_hash[off[p]:off[p + 1]])
    assert (tw.parent >= 0).sum() > win.R // 2      # sessions resend their history: most requests link
    assert tw.chain_off[-1] < win.chain_off[-1] // 2  # and the own blocks are a fraction of the chains


def test_forks_and_unrelated_requests():
    """A request whose session's latest request is not a prefix (a fork) links to an older one that
    is, and a request with no prefix in the window keeps its whole chain."""
    toks = np.arange(16 * 40, dtype=np.uint32)
    a = W.chain_from_tokens(toks[:16 * 10])
    b = W.chain_from_tokens(toks[:16 * 20])                                          # extends a
    c = W.chain_from_tokens(np.concatenate([toks[:16 * 10], toks[16 * 30:16 * 35]]))  # forks from a
    d = W.chain_from_tokens(toks[16 * 5:16 * 9])                                      # unrelated
    chains = [a, b, c, d]
    off = np.zeros(5, np.uint64)
    off[1:] = np.cumsum([len(x) for x in chains])
    win = W.Window(chain_off=off, chain_hash=np.concatenate(chains).astype(np.uint64),
                   prompt_tokens=np.array([16 * len(x) for x in chains], np.uint32),
                   ttft_target=np.ones(4, np.float32), tpot_target=np.ones(4, np.float32),
                   session=np.array([7, 7, 7, 7], np.uint32), out_tokens=np.zeros(4, np.uint32))
    tw = W.tree_window(win)
    assert tw.parent.tolist() == [-1, 0, 0, -1]
    assert np.diff(tw.chain_off).tolist() == [10, 10, 5, 4]
    for r, ch in enumerate(_rebuild(tw)):
        assert np.array_equal(ch, chains[r])
