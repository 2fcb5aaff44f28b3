"""Pin of the oracle's leaf-first LRU eviction against a second characterisation of the same rule.

Evicting, again and again, the cached leaf with the smallest (last_use, hash) removes the blocks in
increasing order of their subtree maximum: eff(v) = the largest (last_use, hash) over v and all its
descendants, a block before its ancestors when two share it.  (Every block u with eff(u) < eff(v)
goes before v: while u or a descendant of u is cached, some leaf below u has a key at most eff(u),
so neither v nor the block w below v whose key is eff(v) can be the smallest leaf.  Blocks with one
subtree maximum lie on one root path.)  So the blocks left after evicting E are all but the E
smallest by (eff, deeper first), which these tests compute in Python from the chains alone and
compare with the oracle's sequential eviction on random branching caches.
"""
import numpy as np
import pytest

import workload as W
from oracle import Oracle


def _random_forest(rng, n_families=4, chains_per_family=5):
    """Chains of explicit tokens that share prefixes (a family branches off its earlier chains),
    each with a last_use stamp; returns [(chain hashes, last_use)]."""
    out = []
    for f in range(n_families):
        fam = []
        for c in range(chains_per_family):
            if fam and rng.random() < 0.8:
                base = fam[rng.integers(len(fam))]
                keep = int(rng.integers(0, len(base) // 16 + 1)) * 16
                toks = np.concatenate([base[:keep], rng.integers(0, 131072, size=16 * int(rng.integers(1, 9)))])
            else:
                toks = rng.integers(0, 131072, size=16 * int(rng.integers(1, 12)))
            toks = toks.astype(np.uint32)
            fam.append(toks)
            out.append((W.chain_from_tokens(toks), int(rng.integers(1, 6))))
    return out


def _predicted_survivors(chains, E):
    """The blocks left after E evictions by the subtree-maximum characterisation."""
    parent, last_use, depth = {}, {}, {}
    for ch, lu in chains:
        for k, h in enumerate(int(x) for x in ch):
            parent.setdefault(h, int(ch[k - 1]) if k else None)
            depth[h] = k
            last_use[h] = max(last_use.get(h, 0), lu)
    children = {h: [] for h in parent}
    for h, p in parent.items():
        if p is not None:
            children[p].append(h)
    eff = {}

    def subtree_max(h):  # iterative post-order
        stack = [(h, False)]
        while stack:
            v, done = stack.pop()
            if v in eff:
                continue
            if done:
                eff[v] = max([(last_use[v], v)] + [eff[c] for c in children[v]])
            else:
                stack.append((v, True))
                stack.extend((c, False) for c in children[v] if c not in eff)

    for h in parent:
        subtree_max(h)
    order = sorted(parent, key=lambda v: (eff[v], -depth[v]))
    return set(order[E:]), len(order)


@pytest.mark.parametrize("seed", [0, 1, 2, 3, 4, 5])
def test_eviction_set_matches_subtree_maximum_order(seed):
    rng = np.random.default_rng(seed)
    chains = _random_forest(rng)
    _, total = _predicted_survivors(chains, 0)
    for E in sorted({1, 2, total // 7, total // 3, total // 2, total - 1}):
        if E <= 0 or E >= total:
            continue
        o = Oracle(1, dict(W.MODEL_DEFAULT), track_lru=True)
        o.set_state(np.zeros(1, np.int32), np.zeros(1, np.int32), np.zeros(1, np.int64), np.zeros(1, np.int64),
                    np.full(1, 10 ** 9, np.int64), np.full(1, 64, np.int32))
        for ch, lu in chains:
            o.insert_chain(0, ch, last_use=lu)
        assert o.cached_blocks(0) == total
        o.set_capacity(np.array([total - E], np.uint64))
        o.load_requests(dict(inst=[], state=[], L=[], out=[], rem=[]))
        o.advance(20.0, 0)
        keep, _ = _predicted_survivors(chains, E)
        assert o.cached_blocks(0) == total - E
        for ch, _ in chains:
            for h in (int(x) for x in ch):
                assert o.contains(0, h) == (h in keep), (seed, E, h)


def test_streaming_stamps_are_monotone_and_eviction_takes_whole_windows():
    """Under the streaming rules a commit stamps the whole chain of an admitted request on its
    instance (cached prefix and new blocks) with the window, so along every cached chain a block's
    last_use is at least its child's; with the subtree-maximum order above, eviction then takes
    blocks oldest window first: no evicted block is newer than a surviving one."""
    wl = W.generate(0, seed=5)
    ins = wl.instances
    o = Oracle(ins.I, wl.model, track_lru=True).load(ins)
    o.set_capacity(np.full(ins.I, 1500, np.uint64))  # below the seeded caches: every window evicts
    o.load_requests(dict(inst=[], state=[], L=[], out=[], rem=[]))  # nothing in flight: requests admitted
    tracked = []  # chains of every window so far
    evicted_any = False
    for w in range(4):
        win = wl.window if w == 0 else wl.next_window(24)
        o.schedule(win, window_id=w + 1, streaming=True)
        tracked += [win.chain_hash[win.chain_off[r]:win.chain_off[r + 1]] for r in range(win.R)]
        blocks = {int(h) for ch in tracked for h in ch}
        before = {(i, h): o.last_use(i, h) for i in range(ins.I) for h in blocks if o.contains(i, h)}
        for i in range(ins.I):
            for ch in tracked:
                for k in range(1, len(ch)):
                    if o.contains(i, int(ch[k])):
                        assert o.contains(i, int(ch[k - 1]))
                        assert o.last_use(i, int(ch[k - 1])) >= o.last_use(i, int(ch[k])), (w, i, k)
        o.advance(20.0, 1000)
        for i in range(ins.I):
            gone = [lu for (j, h), lu in before.items() if j == i and not o.contains(i, h)]
            kept = [lu for (j, h), lu in before.items() if j == i and o.contains(i, h)]
            if gone and kept:
                evicted_any = True
                assert max(gone) <= min(kept), (w, i, max(gone), min(kept))
    assert evicted_any
