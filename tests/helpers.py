"""Shared test inputs: the hand-worked example and small seeded windows."""
from __future__ import annotations

import json
import os

import numpy as np

import workload as W

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")

_SEQ = {"A": (7, 3), "B": (11, 5), "D": (13, 1)}


def seq_tokens(name: str, n: int) -> np.ndarray:
    m, c = _SEQ[name]
    k = np.arange(n, dtype=np.int64)
    return ((m * k + c) % 131072).astype(np.uint32)


def hand_example():
    """Instances, window and expected values of tests/golden/hand_example.json."""
    with open(os.path.join(GOLDEN, "hand_example.json")) as f:
        d = json.load(f)
    I = len(d["instances"])
    chains, inst_ids, parents = [], [], []
    for i, s in enumerate(d["instances"]):
        name, nblk = s["cached"]
        ch = W.chain_from_tokens(seq_tokens(name, 16 * nblk))
        chains.append(ch)
        inst_ids.append(i)
        parents.append(0)
    off = np.zeros(len(chains) + 1, np.uint64)
    off[1:] = np.cumsum([c.shape[0] for c in chains])
    ins = W.Instances(
        b=np.array([s["b"] for s in d["instances"]], np.int32),
        qr=np.array([s["qr"] for s in d["instances"]], np.int32),
        q=np.array([s["q"] for s in d["instances"]], np.int64),
        S=np.array([s["S"] for s in d["instances"]], np.int64),
        M_KV=np.array([s["M_KV"] for s in d["instances"]], np.int64),
        B_max=np.array([s["B_max"] for s in d["instances"]], np.int32),
        cap_blocks=np.full(I, 4096, np.uint64),
        chain_inst=np.array(inst_ids, np.uint32), chain_off=off,
        chain_hash=np.concatenate(chains).astype(np.uint64),
        chain_parent=np.array(parents, np.uint64))
    win = make_window([(seq_tokens(r["seq"], r["L"]), r["ttft_target"], r["tpot_target"])
                       for r in d["requests"]])
    return d["model"], ins, win, d


def make_window(reqs) -> W.Window:
    """reqs: list of (tokens, ttft_target, tpot_target)."""
    chains = [W.chain_from_tokens(t) for t, _, _ in reqs]
    off = np.zeros(len(reqs) + 1, np.uint64)
    off[1:] = np.cumsum([c.shape[0] for c in chains])
    R = len(reqs)
    return W.Window(chain_off=off,
                    chain_hash=(np.concatenate(chains).astype(np.uint64) if R else
                                np.zeros(0, np.uint64)),
                    prompt_tokens=np.array([len(t) for t, _, _ in reqs], np.uint32),
                    ttft_target=np.array([a for _, a, _ in reqs], np.float32),
                    tpot_target=np.array([b for _, _, b in reqs], np.float32),
                    session=np.zeros(R, np.uint32), out_tokens=np.zeros(R, np.uint32))


def lcp(a: np.ndarray, b: np.ndarray) -> int:
    n = min(a.shape[0], b.shape[0])
    neq = np.nonzero(a[:n] != b[:n])[0]
    return int(neq[0]) if neq.size else n
