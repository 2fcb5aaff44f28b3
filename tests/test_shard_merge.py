"""Column-block scoring on the CPU: an instance pool split into blocks, each scored by its own oracle,
merged by the library's merge layer (paper_2609_33224_gb300.shard) over gloo ranks.

Algorithm 1 (Section 6) reduces each request's row twice, W_min over A and then the smallest key over
C, so the pool's decision follows from the blocks' partial results: the MIN over blocks of their
W_min, then each block's pick under that W_min, then the smallest of the blocks' picks in the
paper's order.  The expected values are the unsharded oracle's; every block's partial result comes
from an oracle holding only that block's instances (``Oracle.score_rows_block``).

The keys the merge compares are built here from each block's pick, by the order Section 6.2 states
(more decoding requests, more cached blocks, fewer queued requests, lowest id) and the LMetric product
of the fallback: an encoding the test writes out on its own, not the library's.
"""
import os
import socket

import numpy as np
import pytest

import workload as W
from oracle import Oracle
from paper_2609_33224_gb300 import shard

NO_W = 0xFFFFFFFF


def f2ord(x: np.ndarray) -> np.ndarray:
    """Order-preserving u32 bits of fp32 values (negative: all bits flipped; else the sign bit set)."""
    u = np.asarray(x, np.float32).view(np.uint32)
    return np.where(u & np.uint32(0x80000000), ~u, u | np.uint32(0x80000000)).astype(np.uint32)


def ord2f(o: np.ndarray) -> np.ndarray:
    o = np.asarray(o, np.uint32)
    u = np.where(o & np.uint32(0x80000000), o & np.uint32(0x7FFFFFFF), ~o).astype(np.uint32)
    return u.view(np.float32)


def block_key(ins_blk, L, pick, path, hit) -> tuple:
    """(key, tie) of a block's pick: class 0 keyed by (-b, -h, qr), class 1 by (q + n)(b + qr + 1)."""
    if pick < 0:
        return (1 << 64) - 1, NO_W
    b, qr, q = int(ins_blk.b[pick]), int(ins_blk.qr[pick]), int(ins_blk.q[pick])
    if path == 0:
        v = ((2**18 - 1 - b) << 44) | ((2**26 - 1 - int(hit)) << 18) | qr
    else:
        n = int(L) - 16 * int(hit)
        v = (q + n) * (b + qr + 1)
    return (int(path) << 62) | v, pick


def block_partials(wl, lo, hi, rows, allreduce_min):
    """One block's two phases through the merge layer; returns the merged result and the block's
    classes under the pool's W_min."""
    ins_b = W.column_block(wl.instances, lo, hi)
    orc = Oracle(ins_b.I, wl.model).load(ins_b)
    p1 = orc.score_rows_block(wl.window, rows=rows)
    local = np.where(p1["anyA"] != 0, f2ord(p1["wmin"]), np.uint32(NO_W)).astype(np.uint32)
    wpool = shard.pool_wmin(local, allreduce_min).numpy().astype(np.uint32)
    p2 = orc.score_rows_block(wl.window, wmin=ord2f(wpool), rows=rows)
    L = wl.window.prompt_tokens[rows]
    keys, ties = np.zeros(len(rows), np.uint64), np.zeros(len(rows), np.uint32)
    for k in range(len(rows)):
        pk = int(p2["best"][k])
        kk, tt = block_key(ins_b, L[k], pk, p2["path"][k], p2["hits"][k, pk] if pk >= 0 else 0)
        keys[k] = np.uint64(kk)
        ties[k] = np.uint32(tt + lo if pk >= 0 else NO_W)
    merged = shard.merge_picks(keys, ties, wpool.astype(np.int64), allreduce_min)
    orc.close()
    return merged, p2["cls"], wpool


def _cases():
    """(workload, split point): the default window, eta = 0 (C = the longest hits of A) and tight
    TPOT targets (the LMetric fallback decides most rows)."""
    wl0 = W.generate(0)
    wl_tight = W.generate(0)
    wl_tight.model = dict(wl_tight.model, eta=0.0)
    wl_fb = W.generate(0)
    wl_fb.window.tpot_target[:] = np.float32(12.0)  # few instances pass: fallback rows
    return [(wl0, 3), (wl_tight, 5), (wl_fb, 4)]


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        out = []
        for wl, cut in _cases():
            rows = np.arange(wl.window.R, dtype=np.uint32)
            lo, hi = (0, cut) if rank == 0 else (cut, wl.instances.I)
            merged, cls, wpool = block_partials(wl, lo, hi, rows, shard.dist_allreduce_min())
            out.append((merged["best"], merged["path"], cls, lo, hi, wpool))
        q.put((rank, out))
    finally:
        dist.destroy_process_group()


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_two_gloo_ranks_merge_to_the_unsharded_oracle():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = dict(q.get(timeout=240) for _ in range(2))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for c, (wl, cut) in enumerate(_cases()):
        full = Oracle(wl.instances.I, wl.model).load(wl.instances).score_rows(wl.window)
        for rank in (0, 1):
            best, path, cls, lo, hi, wpool = got[rank][c]
            assert np.array_equal(best, full["best"]), (c, rank)
            assert np.array_equal(path, full["path"]), (c, rank)
            assert np.array_equal(cls, full["cls"][:, lo:hi]), (c, rank)
        assert np.array_equal(got[0][c][5], got[1][c][5])  # one pool W_min on every rank
    # the cases reach both selection paths
    paths = np.concatenate([got[0][c][1] for c in range(3)])
    assert (paths == 0).any() and (paths == 1).any()


class _OneRank:
    """allreduce_min over a single block (world size 1): the identity."""
    def __call__(self, t):
        return t


@pytest.mark.parametrize("cut", [1, 4, 7])
def test_block_decomposition_in_one_process(cut):
    """Blocks scored one after the other, merged by hand (the MIN over blocks written out)."""
    wl = W.generate(0)
    I = wl.instances.I
    rows = np.arange(wl.window.R, dtype=np.uint32)
    full = Oracle(I, wl.model).load(wl.instances).score_rows(wl.window)
    blocks = [(0, cut), (cut, I)]
    orcs = [Oracle(hi - lo, wl.model).load(W.column_block(wl.instances, lo, hi)) for lo, hi in blocks]
    p1 = [o.score_rows_block(wl.window) for o in orcs]
    # a block's own W_min is not the pool's: scored alone, some of its pairs change class
    assert sum(int((p["cls"] != full["cls"][:, lo:hi]).sum()) for p, (lo, hi) in zip(p1, blocks)) > 0
    wl_bits = [np.where(p["anyA"] != 0, f2ord(p["wmin"]), np.uint32(NO_W)) for p in p1]
    wpool = np.minimum(*wl_bits).astype(np.uint32)
    cand = []
    for (lo, hi), o in zip(blocks, orcs):
        p2 = o.score_rows_block(wl.window, wmin=ord2f(wpool))
        ins_b = W.column_block(wl.instances, lo, hi)
        cand.append([block_key(ins_b, wl.window.prompt_tokens[k], int(p2["best"][k]), p2["path"][k],
                               p2["hits"][k, p2["best"][k]] if p2["best"][k] >= 0 else 0)
                     for k in range(wl.window.R)])
        cand[-1] = [(kk, tt + lo if tt != NO_W else NO_W) for kk, tt in cand[-1]]
        assert np.array_equal(p2["cls"], full["cls"][:, lo:hi])
    for k in range(wl.window.R):
        kk, tt = min(cand[0][k], cand[1][k])
        want = full["best"][k]
        assert (tt if (kk != (1 << 64) - 1 and wpool[k] != NO_W) else -1) == want, k
    for o in orcs:
        o.close()
    # the merge layer on one block gives back that block's own pick
    o = Oracle(I, wl.model).load(wl.instances)
    p1 = o.score_rows_block(wl.window)
    local = np.where(p1["anyA"] != 0, f2ord(p1["wmin"]), np.uint32(NO_W)).astype(np.uint32)
    wpool = shard.pool_wmin(local, _OneRank()).numpy()
    p2 = o.score_rows_block(wl.window, wmin=ord2f(wpool.astype(np.uint32)))
    keys = np.array([block_key(wl.instances, wl.window.prompt_tokens[k], int(p2["best"][k]), p2["path"][k],
                               p2["hits"][k, p2["best"][k]] if p2["best"][k] >= 0 else 0)[0]
                     for k in range(wl.window.R)], dtype=np.uint64)
    ties = np.where(p2["best"] >= 0, p2["best"].astype(np.int64), NO_W).astype(np.uint32)
    m = shard.merge_picks(keys, ties, wpool, _OneRank())
    assert np.array_equal(m["best"], full["best"]) and np.array_equal(m["path"], full["path"])


def test_order_preserving_bits_round_trip():
    x = np.array([-3.5, -0.0, 0.0, 1e-30, 2.0, 7e5], np.float32)
    o = f2ord(x)
    assert np.all(np.diff(o.astype(np.int64)) >= 0)
    assert np.array_equal(ord2f(o).view(np.uint32), x.view(np.uint32))


def test_thread_ranks_merge_to_the_unsharded_oracle():
    """The same two phases with the blocks as threads of one process (shard.LocalGroup)."""
    import threading
    wl = W.generate(0)
    I = wl.instances.I
    rows = np.arange(wl.window.R, dtype=np.uint32)
    full = Oracle(I, wl.model).load(wl.instances).score_rows(wl.window)
    cuts = [0, 2, 6, I]
    grp = shard.LocalGroup(len(cuts) - 1)
    out, errs = [None] * (len(cuts) - 1), []

    def work(k):
        try:
            out[k] = block_partials(wl, cuts[k], cuts[k + 1], rows, grp.allreduce_min(k))
        except BaseException as e:  # noqa: BLE001 - reported below
            errs.append(e)
            grp.abort()

    th = [threading.Thread(target=work, args=(k,)) for k in range(len(cuts) - 1)]
    for t in th:
        t.start()
    for t in th:
        t.join(timeout=120)
    assert not errs, errs
    for k, (merged, cls, _) in enumerate(out):
        assert np.array_equal(merged["best"], full["best"]) and np.array_equal(merged["path"], full["path"])
        assert np.array_equal(cls, full["cls"][:, cuts[k]:cuts[k + 1]])


def test_blocks_without_capacity_and_rows_rejected_everywhere():
    """Edge cases of the merge, blocks as threads: the first block has no instance with a free
    decode slot (b + qr + 1 > B_max), so its W_min and its key are the 'none' values on every row,
    and the second block's KV room fits only the shorter prompts (S + L <= M_KV), so the longer
    requests pass the capacity guard nowhere and are rejected (Algorithm 1: A empty)."""
    import threading
    wl = W.generate(0)
    ins = wl.instances
    cut = 3
    ins.b[:cut] = ins.B_max[:cut]
    med = int(np.median(wl.window.prompt_tokens))
    ins.M_KV[cut:] = ins.S[cut:] + med
    I = ins.I
    full = Oracle(I, wl.model).load(ins).score_rows(wl.window)
    assert (full["best"] < 0).any() and (full["best"] >= 0).any()
    assert (full["best"][full["best"] >= 0] >= cut).all()
    rows = np.arange(wl.window.R, dtype=np.uint32)
    cuts = [0, cut, I]
    grp = shard.LocalGroup(2)
    out, errs = [None, None], []

    def work(k):
        try:
            out[k] = block_partials(wl, cuts[k], cuts[k + 1], rows, grp.allreduce_min(k))
        except BaseException as e:  # noqa: BLE001 - reported below
            errs.append(e)
            grp.abort()

    th = [threading.Thread(target=work, args=(k,)) for k in range(2)]
    for t in th:
        t.start()
    for t in th:
        t.join(timeout=120)
    assert not errs, errs
    for k, (merged, cls, wpool) in enumerate(out):
        assert np.array_equal(merged["best"], full["best"]), k
        assert np.array_equal(merged["path"], full["path"]), k
        assert np.array_equal(cls, full["cls"][:, cuts[k]:cuts[k + 1]]), k
    # a row rejected everywhere has no pool W_min at all
    rej = full["best"] < 0
    assert (out[0][2][rej] == np.uint32(NO_W)).all()
