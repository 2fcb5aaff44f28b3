"""Python handle on the oracle (TEST INFRASTRUCTURE).

The oracle is a plain single-threaded C++ restatement of the paper's Algorithm 1 (see the header
of ``ps_oracle.cpp``).  Only the tests, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline
and reference legs may import this package; the product library never does.

Parity status of each oracle function (what pins it, in ``tests/test_oracle_pins.py``):
  * hit length           -- brute-force token longest-common-prefix on explicit token lists.
  * T_pf / W / Z / rho   -- closed forms under the workload coefficients, fp64 cross-check.
  * TPOT / TTFT          -- hand-computed literals (golden hand example), fp64 cross-check.
  * filters and picks    -- special cases of Sections 6.1/6.2 (eta = 0, Z = 0, T empty, A empty),
                            exhaustive brute force over tiny instance sets.
  * greedy               -- hand-traced tiny windows; replay invariant (each decision equals the
                            single-request rule on the state left by the earlier decisions).
  * policy variants      -- Table 3 ablations and Table 4 selectors on a hand-worked request
                            (``tests/test_oracle_policies.py``).
  * online calibration   -- hand trace, closed form of a constant ratio, bounds
                            (``tests/test_oracle_calibration.py``).
  * eviction             -- hand traces, and the evicted set against the subtree-maximum order on
                            random branching caches (``tests/test_oracle_eviction_order.py``).
No oracle function is left "parity unpinned".
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "libps_oracle.so")
_LOCK = threading.Lock()
_LIB = None

INST_DTYPE = np.dtype([("b", np.int32), ("qr", np.int32), ("q", np.int64), ("S", np.int64),
                       ("M_KV", np.int64), ("B_max", np.int32)], align=True)


class OrcModel(ctypes.Structure):
    _fields_ = [(k, ctypes.c_float) for k in
                ("a0", "a1", "a2", "a3", "a4", "a5", "b0", "b1", "b2", "g_q", "eta", "lout_median")] + [
        ("interference_mode", ctypes.c_int32), ("ttft_filter", ctypes.c_int32),
        ("nseg", ctypes.c_int32), ("seg_lo", ctypes.c_int32 * 16), ("ema_factor", ctypes.c_float * 16),
        ("cache_filter", ctypes.c_int32), ("slo_filter", ctypes.c_int32), ("fallback", ctypes.c_int32),
        ("selector", ctypes.c_int32)]

# Instance orders inside T (Table 4) and the ablation configurations (Table 3) as model keys.
SELECTORS = {"D-C-Q": 0, "D": 1, "D-Q": 2, "D-C": 3, "D-Q-C": 4, "H-C-Q": 5}
ABLATIONS = {"G": dict(cache_filter=0, slo_filter=0, fallback=1), "C": dict(cache_filter=1, slo_filter=0, fallback=1),
             "T": dict(cache_filter=0, slo_filter=1, fallback=1), "CT": dict(cache_filter=1, slo_filter=1, fallback=1),
             "F": dict(cache_filter=1, slo_filter=1, fallback=0)}


def build(force: bool = False) -> str:
    """Compile the oracle: -O2 -ffp-contract=off so no multiply-add is ever fused."""
    with _LOCK:
        src = os.path.join(_HERE, "ps_oracle.cpp")
        if not force and os.path.exists(_SO) and os.path.getmtime(_SO) >= os.path.getmtime(src):
            return _SO
        os.makedirs(_BUILD, exist_ok=True)
        tmp = _SO + f".tmp{os.getpid()}"
        subprocess.run(["g++", "-O2", "-std=c++17", "-ffp-contract=off", "-fno-fast-math",
                        "-fPIC", "-shared", "-o", tmp, src], check=True)
        os.replace(tmp, _SO)
        return _SO


def _lib():
    global _LIB
    if _LIB is None:
        lib = ctypes.CDLL(build())
        vp, u32, u64, i32 = ctypes.c_void_p, ctypes.c_uint32, ctypes.c_uint64, ctypes.c_int32
        lib.orc_create.restype = vp
        lib.orc_create.argtypes = [u32, ctypes.POINTER(OrcModel), i32]
        lib.orc_destroy.argtypes = [vp]
        lib.orc_reserve.argtypes = [vp, u32, u64]
        lib.orc_insert_chain.argtypes = [vp, u32, vp, u64, u64, u32]
        lib.orc_insert_chains.argtypes = [vp, u64, vp, vp, vp, vp, u32]
        lib.orc_cached_blocks.restype = u64
        lib.orc_cached_blocks.argtypes = [vp, u32]
        lib.orc_contains.restype = i32
        lib.orc_contains.argtypes = [vp, u32, u64]
        lib.orc_set_state.argtypes = [vp, vp]
        lib.orc_get_state.argtypes = [vp, vp]
        lib.orc_hit.restype = u64
        lib.orc_hit.argtypes = [vp, u32, vp, u64]
        lib.orc_hit_pairs.argtypes = [vp, vp, vp, u64, vp, vp, vp]
        lib.orc_score_rows.argtypes = [vp] * 6 + [u64] + [vp] * 7
        lib.orc_score_rows_block.argtypes = [vp] * 6 + [u64] + [vp] * 8
        lib.orc_schedule.argtypes = [vp, u32] + [vp] * 9 + [u32]
        lib.orc_set_capacity.argtypes = [vp, vp]
        lib.orc_load_requests.argtypes = [vp, u64, vp, vp, vp, vp, vp]
        lib.orc_advance.argtypes = [vp, ctypes.c_float, u64, i32]
        lib.orc_last_use.restype = u32
        lib.orc_last_use.argtypes = [vp, u32, u64]
        lib.orc_calibrate.argtypes = [vp, u64, vp, vp, vp, ctypes.c_float]
        lib.orc_ema_factors.argtypes = [vp, vp]
        _LIB = lib
    return _LIB


def _p(a):
    return None if a is None else a.ctypes.data


def make_model(model: dict) -> OrcModel:
    m = OrcModel()
    for k in ("a0", "a1", "a2", "a3", "a4", "a5", "b0", "b1", "b2", "g_q", "eta", "lout_median"):
        setattr(m, k, float(model[k]))
    m.interference_mode = int(model.get("interference_mode", 0))
    m.ttft_filter = int(model.get("ttft_filter", 1))
    seg_lo = list(model.get("seg_lo", [0]))
    ema = list(model.get("ema_factor", [1.0]))
    if not (1 <= len(seg_lo) <= 16) or len(ema) != len(seg_lo):
        raise ValueError("EMA segments: 1..16 lower bounds with one factor each")
    m.nseg = len(seg_lo)
    for k, (lo, f) in enumerate(zip(seg_lo, ema)):
        m.seg_lo[k] = int(lo)
        m.ema_factor[k] = float(f)
    m.cache_filter = int(model.get("cache_filter", 1))
    m.slo_filter = int(model.get("slo_filter", 1))
    m.fallback = int(model.get("fallback", 0))
    m.selector = int(model.get("selector", 0))
    if m.fallback not in (0, 1) or not 0 <= m.selector <= 5:
        raise ValueError("fallback 0 (LMetric) or 1 (D-C-Q); selector 0..5")
    return m


def _c(a, dt):
    return np.ascontiguousarray(a, dtype=dt)


class Oracle:
    """One oracle scheduler over I instances."""

    def __init__(self, I: int, model: dict, track_lru: bool = False):
        self.I = int(I)
        self.track_lru = bool(track_lru)
        self._m = make_model(model)
        self._h = _lib().orc_create(self.I, ctypes.byref(self._m), 1 if track_lru else 0)
        if not self._h:
            raise ValueError("oracle: invalid model")

    def close(self):
        if self._h:
            _lib().orc_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- instances ---------------------------------------------------------------------------
    def insert_chain(self, inst: int, chain, parent: int = 0, last_use: int = 0):
        c = _c(chain, np.uint64)
        _lib().orc_insert_chain(self._h, int(inst), _p(c), c.shape[0], int(parent), int(last_use))

    def insert_chains(self, inst, off, hash_, parent, last_use: int = 0):
        inst, off = _c(inst, np.uint32), _c(off, np.uint64)
        hash_, parent = _c(hash_, np.uint64), _c(parent, np.uint64)
        _lib().orc_insert_chains(self._h, inst.shape[0], _p(inst), _p(off), _p(hash_), _p(parent),
                                 int(last_use))

    def cached_blocks(self, inst: int) -> int:
        return int(_lib().orc_cached_blocks(self._h, int(inst)))

    def contains(self, inst: int, block: int) -> bool:
        return bool(_lib().orc_contains(self._h, int(inst), int(block)))

    def set_state(self, b, qr, q, S, M_KV, B_max):
        s = np.zeros(self.I, INST_DTYPE)
        s["b"], s["qr"], s["q"], s["S"], s["M_KV"], s["B_max"] = b, qr, q, S, M_KV, B_max
        _lib().orc_set_state(self._h, _p(s))

    def get_state(self) -> dict:
        s = np.zeros(self.I, INST_DTYPE)
        _lib().orc_get_state(self._h, _p(s))
        return {k: s[k].copy() for k in INST_DTYPE.names}

    def load(self, inst) -> "Oracle":
        """Seed caches and state from a workload.Instances (and capacities for eviction)."""
        counts = np.bincount(inst.chain_inst, weights=np.diff(inst.chain_off).astype(np.float64),
                             minlength=self.I)
        for i in range(self.I):
            _lib().orc_reserve(self._h, i, int(counts[i]))
        self.insert_chains(inst.chain_inst, inst.chain_off, inst.chain_hash, inst.chain_parent)
        self.set_state(inst.b, inst.qr, inst.q, inst.S, inst.M_KV, inst.B_max)
        self.set_capacity(inst.cap_blocks)
        return self

    # -- scheduling --------------------------------------------------------------------------
    def hit(self, inst: int, chain) -> int:
        c = _c(chain, np.uint64)
        return int(_lib().orc_hit(self._h, int(inst), _p(c), c.shape[0]))

    def hit_pairs(self, window, req, inst) -> np.ndarray:
        req, inst = _c(req, np.uint32), _c(inst, np.uint32)
        out = np.zeros(req.shape[0], np.uint32)
        _lib().orc_hit_pairs(self._h, _p(_c(window.chain_off, np.uint64)),
                             _p(_c(window.chain_hash, np.uint64)), req.shape[0], _p(req), _p(inst),
                             _p(out))
        return out

    def score_rows(self, window, rows=None) -> dict:
        rows = np.arange(window.R, dtype=np.uint32) if rows is None else _c(rows, np.uint32)
        n = rows.shape[0]
        out = dict(hits=np.zeros((n, self.I), np.uint32), tpot=np.zeros((n, self.I), np.float32),
                   ttft=np.zeros((n, self.I), np.float32), cls=np.zeros((n, self.I), np.uint8),
                   best=np.zeros(n, np.int32), path=np.zeros(n, np.uint8))
        _lib().orc_score_rows(self._h, _p(_c(window.chain_off, np.uint64)),
                              _p(_c(window.chain_hash, np.uint64)),
                              _p(_c(window.prompt_tokens, np.uint32)),
                              _p(_c(window.ttft_target, np.float32)),
                              _p(_c(window.tpot_target, np.float32)), n, _p(rows),
                              _p(out["hits"]), _p(out["tpot"]), _p(out["ttft"]), _p(out["cls"]),
                              _p(out["best"]), _p(out["path"]))
        return out

    def score_rows_block(self, window, wmin=None, rows=None) -> dict:
        """Score mode when this oracle holds one column block of a larger instance pool: returns the
        block's W_min over A ("wmin", valid where "anyA") and, with ``wmin`` given (the pool's W_min
        per row), classes and the block's pick under that W_min (block-local ids)."""
        rows = np.arange(window.R, dtype=np.uint32) if rows is None else _c(rows, np.uint32)
        n = rows.shape[0]
        win = None if wmin is None else _c(wmin, np.float32)
        out = dict(wmin=np.zeros(n, np.float32), anyA=np.zeros(n, np.uint8),
                   hits=np.zeros((n, self.I), np.uint32), cls=np.zeros((n, self.I), np.uint8),
                   best=np.zeros(n, np.int32), path=np.zeros(n, np.uint8))
        _lib().orc_score_rows_block(self._h, _p(_c(window.chain_off, np.uint64)),
                                    _p(_c(window.chain_hash, np.uint64)),
                                    _p(_c(window.prompt_tokens, np.uint32)),
                                    _p(_c(window.ttft_target, np.float32)),
                                    _p(_c(window.tpot_target, np.float32)), n, _p(rows), _p(win),
                                    _p(out["wmin"]), _p(out["anyA"]), _p(out["hits"]), _p(out["cls"]),
                                    _p(out["best"]), _p(out["path"]))
        return out

    def schedule(self, window, window_id: int = 0, streaming: bool = False) -> dict:
        """Greedy window; with streaming=True admitted requests join their instance's queue."""
        R = window.R
        out = dict(assign=np.zeros(R, np.int32), path=np.zeros(R, np.uint8),
                   hit_chosen=np.zeros(R, np.uint32))
        outs = _c(window.out_tokens, np.uint32) if streaming else None
        _lib().orc_schedule(self._h, R, _p(_c(window.chain_off, np.uint64)),
                            _p(_c(window.chain_hash, np.uint64)),
                            _p(_c(window.prompt_tokens, np.uint32)),
                            _p(_c(window.ttft_target, np.float32)),
                            _p(_c(window.tpot_target, np.float32)), _p(outs), _p(out["assign"]),
                            _p(out["path"]), _p(out["hit_chosen"]), int(window_id))
        return out

    # -- streaming windows ---------------------------------------------------------------------
    def set_capacity(self, cap):
        c = _c(cap, np.uint64)
        _lib().orc_set_capacity(self._h, _p(c))

    def load_requests(self, req: dict):
        """req: inst, state (0 queued / 1 decoding), L, out, rem arrays (queued in FIFO order)."""
        inst, state = _c(req["inst"], np.uint32), _c(req["state"], np.uint32)
        L, out, rem = _c(req["L"], np.uint32), _c(req["out"], np.uint32), _c(req["rem"], np.uint64)
        _lib().orc_load_requests(self._h, inst.shape[0], _p(inst), _p(state), _p(L), _p(out), _p(rem))

    def advance(self, window_ms: float = 20.0, prefill_tokens: int = 1000, evict: bool = True):
        _lib().orc_advance(self._h, float(window_ms), int(prefill_tokens), 1 if evict else 0)

    def last_use(self, inst: int, block: int) -> int:
        return int(_lib().orc_last_use(self._h, int(inst), int(block)))

    # -- online calibration (Section 5.3) --------------------------------------------------------
    def calibrate(self, batch, ctx_tokens, measured_ms, weight: float = 0.02):
        """Feed pure-decode samples (batch size, total context tokens, measured ms), in order."""
        b = _c(batch, np.int32)
        c = _c(ctx_tokens, np.int64)
        t = _c(measured_ms, np.float32)
        if not (b.shape == c.shape == t.shape):
            raise ValueError("one batch size, context and duration per sample")
        _lib().orc_calibrate(self._h, b.shape[0], _p(b), _p(c), _p(t), float(weight))

    def ema_factors(self) -> np.ndarray:
        out = np.zeros(16, np.float32)
        _lib().orc_ema_factors(self._h, _p(out))
        return out[: self._m.nseg].copy()
