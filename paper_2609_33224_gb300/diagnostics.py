"""Recompute-budget sweep (Section 8, "Impact of the Recomputation Budget"; Fig. 10 (a)-(b)): how
eta of Eq. 8 trades placement flexibility (the size of the cache-admissible set C) against cache
locality (the KV-cache hit rate of the chosen placements).

For each eta the same window is scheduled once on the same committed state (each
``schedule_window`` leaves a pending window that the next one discards), through the library:
- mean |C| (and |T|) come from the window's independent scores against the committed state
  (``cls`` of ``ps_schedule_window``'s optional scores), averaged over the requests that have a
  capacity-eligible instance;
- the hit rate comes from the greedy decisions: cached prompt tokens of the admitted requests on
  their chosen instances at decision time, over their prompt tokens.
The paper measures both over a replay of its production trace; a synthetic window stands in here.
"""
from __future__ import annotations

import numpy as np

BLOCK_TOKENS = 16
# the paper's sweep: eta from 0 to 1 in steps of 0.1
PAPER_ETAS = tuple(k / 10 for k in range(11))


def window_stats(cls, path, hit_chosen, prompt_tokens) -> dict:
    """Statistics of one scheduling of a window.

    cls: u8[R, I] classes of the independent scores (0 in T, 1 in C outside T, 2 in A outside C,
    3 outside A); path: u8[R] greedy paths (0 packed, 1 fallback, 2 reject); hit_chosen: u32[R]
    hit length in blocks on the chosen instance; prompt_tokens: u32[R].
    """
    cls = np.asarray(cls)
    path = np.asarray(path)
    hit = np.asarray(hit_chosen, np.int64)
    L = np.asarray(prompt_tokens, np.int64)
    R = int(path.shape[0])
    eligible = (cls <= 2).any(axis=1) if cls.size else np.zeros(R, bool)
    c_size = (cls <= 1).sum(axis=1) if cls.size else np.zeros(R, np.int64)
    t_size = (cls == 0).sum(axis=1) if cls.size else np.zeros(R, np.int64)
    admitted = path < 2
    cached = int((BLOCK_TOKENS * hit[admitted]).sum())
    tokens = int(L[admitted].sum())
    n_el = int(eligible.sum())
    return dict(
        requests=R,
        mean_C=float(c_size[eligible].mean()) if n_el else 0.0,
        mean_T=float(t_size[eligible].mean()) if n_el else 0.0,
        packed=int((path == 0).sum()),
        fallback=int((path == 1).sum()),
        rejected=int((path == 2).sum()),
        cached_tokens=cached,
        admitted_tokens=tokens,
        hit_rate=cached / tokens if tokens else 0.0,
    )


def eta_sweep(sched, window, model: dict, etas=PAPER_ETAS) -> list:
    """One greedy scheduling of ``window`` per eta (all else as ``model``), on ``sched``'s committed
    state; the model is restored afterwards.  The last scheduling stays pending, like any other
    (the next ``schedule_window`` or ``load_instances`` discards it).  ``sched`` is a
    ``Scheduler`` (or an object with the same ``set_model`` / ``schedule_window`` methods).
    Returns one ``window_stats`` dict per eta, with its ``eta``."""
    out = []
    try:
        for eta in etas:
            if not eta >= 0.0:
                raise ValueError("eta must be >= 0 (Eq. 8)")
            sched.set_model(dict(model, eta=float(eta)))
            d = sched.schedule_window(window, scores=("cls",))
            st = window_stats(d["scores"]["cls"], d["path"], d["hit_chosen"], window.prompt_tokens)
            st["eta"] = float(eta)
            out.append(st)
    finally:
        sched.set_model(model)
    return out
