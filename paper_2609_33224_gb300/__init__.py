"""Python binding of the GB300 PackServe scheduler library (include/packserve.h).

Argument marshalling only: every step of the hot path (hit lengths, latency model, filters,
argmin, greedy assignment) runs in the CUDA kernels of ``libpackserve.so``.  The raw entry points
keep the C names (``ps_create``, ``ps_score_window`` ...); ``Scheduler`` wraps one context and
accepts numpy arrays (host memory) or CUDA torch tensors (device memory).

The library must be built first (``paper_2609_33224_gb300.build.build()`` or
``__graft_entry__.build()``); importing the binding without it raises, there is no CPU path.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from .build import LIB as _LIB_PATH, build  # noqa: F401

PS_OK, PS_ERR_INVALID, PS_ERR_CUDA, PS_ERR_OOM, PS_ERR_TABLE_FULL, PS_ERR_TIMEOUT, PS_ERR_CAPACITY, \
    PS_ERR_STATE = range(8)
STATUS_NAMES = {0: "PS_OK", 1: "PS_ERR_INVALID", 2: "PS_ERR_CUDA", 3: "PS_ERR_OOM",
                4: "PS_ERR_TABLE_FULL", 5: "PS_ERR_TIMEOUT", 6: "PS_ERR_CAPACITY", 7: "PS_ERR_STATE"}

ABI_FUNCTIONS = ("ps_create", "ps_load_instances", "ps_get_instances", "ps_get_pending_instances",
                 "ps_calibrate", "ps_get_ema_factors", "ps_set_model", "ps_set_wait_limit",
                 "ps_insert_blocks", "ps_insert_chains", "ps_cached_blocks", "ps_score_window",
                 "ps_schedule_window", "ps_commit_window", "ps_last_timings", "ps_last_probe_stats", "ps_last_error",
                 "ps_destroy", "ps_score_window_noalloc", "ps_load_requests", "ps_advance_window",
                 "ps_shard_wmin", "ps_shard_pick")


class PsModel(ctypes.Structure):
    _fields_ = [(k, ctypes.c_float) for k in
                ("a0", "a1", "a2", "a3", "a4", "a5", "b0", "b1", "b2", "g_q", "eta", "lout_median")] + [
        ("interference_mode", ctypes.c_int32), ("ttft_filter", ctypes.c_int32), ("nseg", ctypes.c_int32),
        ("seg_lo", ctypes.c_int32 * 16), ("ema_factor", ctypes.c_float * 16),
        ("cache_filter_off", ctypes.c_int32), ("slo_filter_off", ctypes.c_int32), ("fallback_dcq", ctypes.c_int32),
        ("selector", ctypes.c_int32)]


# Table 4 instance orders (ps_model.selector) and Table 3 admission ablations (ps_model switches).
SELECTORS = {"D-C-Q": 0, "D": 1, "D-Q": 2, "D-C": 3, "D-Q-C": 4, "H-C-Q": 5}
ABLATIONS = {"G": dict(cache_filter_off=1, slo_filter_off=1, fallback_dcq=1),
             "C": dict(cache_filter_off=0, slo_filter_off=1, fallback_dcq=1),
             "T": dict(cache_filter_off=1, slo_filter_off=0, fallback_dcq=1),
             "CT": dict(cache_filter_off=0, slo_filter_off=0, fallback_dcq=1),
             "F": dict(cache_filter_off=0, slo_filter_off=0, fallback_dcq=0)}


class PsConfig(ctypes.Structure):
    _fields_ = [("device", ctypes.c_int32), ("cuda_stream", ctypes.c_void_p),
                ("num_instances", ctypes.c_uint32), ("max_window_requests", ctypes.c_uint32),
                ("max_window_chain_blocks", ctypes.c_uint64), ("block_tokens", ctypes.c_uint32),
                ("cap_blocks", ctypes.c_void_p), ("table_load_factor", ctypes.c_float),
                ("model", PsModel), ("probe_mode", ctypes.c_int32), ("track_lru", ctypes.c_int32),
                ("max_active_requests", ctypes.c_uint32)]

PS_PROBE_LINEAR, PS_PROBE_SEARCH = 0, 1


class PsInstanceState(ctypes.Structure):
    _fields_ = [("b", ctypes.c_int32), ("qr", ctypes.c_int32), ("q_tokens", ctypes.c_int64),
                ("S_tokens", ctypes.c_int64), ("M_KV_tokens", ctypes.c_int64), ("B_max", ctypes.c_int32)]


class PsWindow(ctypes.Structure):
    _fields_ = [("R", ctypes.c_uint32), ("chain_off", ctypes.c_void_p), ("chain_hash", ctypes.c_void_p),
                ("prompt_tokens", ctypes.c_void_p), ("ttft_target", ctypes.c_void_p),
                ("tpot_target", ctypes.c_void_p), ("out_tokens", ctypes.c_void_p),
                ("inputs_on_device", ctypes.c_int32), ("parent", ctypes.c_void_p)]


class PsScores(ctypes.Structure):
    _fields_ = [("hits", ctypes.c_void_p), ("tpot", ctypes.c_void_p), ("ttft", ctypes.c_void_p),
                ("cls", ctypes.c_void_p), ("best", ctypes.c_void_p), ("path", ctypes.c_void_p),
                ("outputs_on_device", ctypes.c_int32)]


class PsDecisions(ctypes.Structure):
    _fields_ = [("assign", ctypes.c_void_p), ("path", ctypes.c_void_p), ("hit_chosen", ctypes.c_void_p),
                ("outputs_on_device", ctypes.c_int32)]


class PsAdvanceParams(ctypes.Structure):
    _fields_ = [("window_ms", ctypes.c_float), ("prefill_tokens", ctypes.c_uint64), ("evict", ctypes.c_int32)]


class PsTableDesc(ctypes.Structure):
    _fields_ = [("base", ctypes.c_uint64), ("overflow_base", ctypes.c_uint64), ("num_buckets", ctypes.c_uint32),
                ("reserved", ctypes.c_uint32)]


class PsStateArrays(ctypes.Structure):
    _fields_ = [(k, ctypes.c_void_p) for k in ("b", "qr", "q_tokens", "S_tokens", "M_KV_tokens", "B_max")]


PS_NOALLOC_MAX_PAIRS = 2097152

STATE_DTYPE = np.dtype([("b", np.int32), ("qr", np.int32), ("q_tokens", np.int64), ("S_tokens", np.int64),
                        ("M_KV_tokens", np.int64), ("B_max", np.int32)], align=True)
assert STATE_DTYPE.itemsize == ctypes.sizeof(PsInstanceState)

_lib = None


def lib() -> ctypes.CDLL:
    """The loaded library; raises if it has not been built (no fallback path exists)."""
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError(f"{_LIB_PATH} is missing: build the CUDA library first "
                               "(python -c 'import __graft_entry__ as g; g.build()')")
        L = ctypes.CDLL(_LIB_PATH)
        vp, u32, u64, i32, st = ctypes.c_void_p, ctypes.c_uint32, ctypes.c_uint64, ctypes.c_int32, ctypes.c_int
        sigs = {
            "ps_create": [ctypes.POINTER(PsConfig), ctypes.POINTER(vp)],
            "ps_load_instances": [vp, vp, u32],
            "ps_get_instances": [vp, vp, u32],
            "ps_get_pending_instances": [vp, vp, u32],
            "ps_insert_blocks": [vp, u32, vp, u64, u64, u32],
            "ps_insert_chains": [vp, u64, vp, vp, vp, vp, u32, i32],
            "ps_cached_blocks": [vp, vp, u32],
            "ps_score_window": [vp, ctypes.POINTER(PsWindow), ctypes.POINTER(PsScores)],
            "ps_schedule_window": [vp, ctypes.POINTER(PsWindow), ctypes.POINTER(PsDecisions),
                                   ctypes.POINTER(PsScores)],
            "ps_commit_window": [vp, u32],
            "ps_last_timings": [vp, vp, u32],
            "ps_last_probe_stats": [vp, vp, u32],
            "ps_calibrate": [vp, u32, vp, vp, vp, ctypes.c_float],
            "ps_get_ema_factors": [vp, vp, u32],
            "ps_set_model": [vp, ctypes.POINTER(PsModel)],
            "ps_set_wait_limit": [vp, u64],
            "ps_load_requests": [vp, u64, vp, vp, vp, vp, vp],
            "ps_advance_window": [vp, ctypes.POINTER(PsAdvanceParams)],
            "ps_shard_wmin": [vp, ctypes.POINTER(PsWindow), vp, i32],
            "ps_shard_pick": [vp, vp, u32, vp, vp, i32, ctypes.POINTER(PsScores)],
            "ps_score_window_noalloc": [vp, vp, vp, u32, ctypes.POINTER(PsStateArrays), ctypes.POINTER(PsWindow),
                                        ctypes.POINTER(PsModel), i32, ctypes.POINTER(PsScores), vp],
        }
        for name, args in sigs.items():
            fn = getattr(L, name)
            fn.argtypes = args
            fn.restype = st
        L.ps_last_error.argtypes = [vp]
        L.ps_last_error.restype = ctypes.c_char_p
        L.ps_destroy.argtypes = [vp]
        L.ps_destroy.restype = None
        _lib = L
    return _lib


def __getattr__(name):  # ps_* names resolve to the C entry points
    if name in ABI_FUNCTIONS:
        return getattr(lib(), name)
    raise AttributeError(name)


class PSError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


def make_model(model: dict) -> PsModel:
    m = PsModel()
    for k in ("a0", "a1", "a2", "a3", "a4", "a5", "b0", "b1", "b2", "g_q", "eta", "lout_median"):
        setattr(m, k, float(model[k]))
    m.interference_mode = int(model.get("interference_mode", 0))
    m.ttft_filter = int(model.get("ttft_filter", 1))
    seg_lo = list(model.get("seg_lo", [0]))
    ema = list(model.get("ema_factor", [1.0]))
    m.nseg = len(seg_lo)
    for k, (lo, f) in enumerate(zip(seg_lo, ema)):
        m.seg_lo[k] = int(lo)
        m.ema_factor[k] = float(f)
    for k in ("cache_filter_off", "slo_filter_off", "fallback_dcq", "selector"):
        setattr(m, k, int(model.get(k, 0)))
    return m


def _is_torch(x) -> bool:
    return type(x).__module__.startswith("torch")


def _ptr(x, dtype=None):
    """(pointer, on_device) of a numpy array or torch tensor; None -> (None, None)."""
    if x is None:
        return None, None
    if _is_torch(x):
        if not x.is_contiguous():
            raise ValueError("tensors must be contiguous")
        return (x.data_ptr() if x.numel() else None), bool(x.is_cuda)
    if dtype is not None and (x.dtype != dtype or not x.flags["C_CONTIGUOUS"]):
        raise ValueError(f"expected a contiguous {np.dtype(dtype)} array, got {x.dtype}")
    return (x.ctypes.data if x.size else None), False


class Scheduler:
    """One scheduler context on one GPU (``ps_create`` ... ``ps_destroy``)."""

    def __init__(self, num_instances: int, cap_blocks, max_window_requests: int,
                 max_window_chain_blocks: int, model: dict, table_load_factor: float = 0.5,
                 device: int = 0, stream=None, probe_mode: int = PS_PROBE_SEARCH, track_lru: bool = False,
                 max_active_requests: int = 0):
        self.I = int(num_instances)
        self._cap = np.ascontiguousarray(cap_blocks, dtype=np.uint64)
        cfg = PsConfig()
        cfg.device = int(device)
        cfg.cuda_stream = stream
        cfg.num_instances = self.I
        cfg.max_window_requests = int(max_window_requests)
        cfg.max_window_chain_blocks = int(max_window_chain_blocks)
        cfg.block_tokens = 16
        cfg.cap_blocks = self._cap.ctypes.data
        cfg.table_load_factor = float(table_load_factor)
        cfg.model = make_model(model)
        self.selector = int(cfg.model.selector)  # the instance order inside T (Table 4)
        cfg.probe_mode = int(probe_mode)
        cfg.track_lru = 1 if track_lru else 0
        cfg.max_active_requests = int(max_active_requests)
        self.probe_mode = int(probe_mode)
        h = ctypes.c_void_p()
        s = lib().ps_create(ctypes.byref(cfg), ctypes.byref(h))
        if s != PS_OK:
            raise PSError(s, "ps_create failed (invalid configuration or device allocation)")
        self._h = h
        self.device = int(device)

    # ------------------------------------------------------------------------------------------
    def _check(self, s: int):
        if s != PS_OK:
            raise PSError(s, lib().ps_last_error(self._h).decode())

    def close(self):
        if getattr(self, "_h", None):
            lib().ps_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *a):
        self.close()

    @property
    def handle(self):
        return self._h

    # ------------------------------------------------------------------------------------------
    def load_instances(self, b, qr, q, S, M_KV, B_max):
        st = np.zeros(self.I, STATE_DTYPE)
        st["b"], st["qr"], st["q_tokens"], st["S_tokens"] = b, qr, q, S
        st["M_KV_tokens"], st["B_max"] = M_KV, B_max
        self._check(lib().ps_load_instances(self._h, st.ctypes.data, self.I))

    def load_workload_instances(self, ins):
        """Seed caches and state from a workload.Instances-like object."""
        self.insert_chains(ins.chain_inst, ins.chain_off, ins.chain_hash, ins.chain_parent)
        self.load_instances(ins.b, ins.qr, ins.q, ins.S, ins.M_KV, ins.B_max)

    def get_instances(self, pending: bool = False) -> dict:
        st = np.zeros(self.I, STATE_DTYPE)
        fn = lib().ps_get_pending_instances if pending else lib().ps_get_instances
        self._check(fn(self._h, st.ctypes.data, self.I))
        return {"b": st["b"].copy(), "qr": st["qr"].copy(), "q": st["q_tokens"].copy(),
                "S": st["S_tokens"].copy(), "M_KV": st["M_KV_tokens"].copy(), "B_max": st["B_max"].copy()}

    def insert_blocks(self, inst: int, chain, parent: int = 0, last_use: int = 0):
        c = np.ascontiguousarray(chain, dtype=np.uint64)
        self._check(lib().ps_insert_blocks(self._h, int(inst), c.ctypes.data if c.size else None, c.size,
                                           int(parent), int(last_use)))

    def insert_chains(self, inst, off, hash_, parent, last_use: int = 0):
        if _is_torch(off):
            args = [_ptr(x)[0] for x in (inst, off, hash_, parent)]
            n = int(off.numel()) - 1
            self._check(lib().ps_insert_chains(self._h, n, *args, int(last_use), 1))
            return
        inst = np.ascontiguousarray(inst, np.uint32)
        off = np.ascontiguousarray(off, np.uint64)
        hash_ = np.ascontiguousarray(hash_, np.uint64)
        parent = np.ascontiguousarray(parent, np.uint64)
        self._check(lib().ps_insert_chains(self._h, inst.shape[0], inst.ctypes.data, off.ctypes.data,
                                           hash_.ctypes.data if hash_.size else None, parent.ctypes.data,
                                           int(last_use), 0))

    def cached_blocks(self) -> np.ndarray:
        out = np.zeros(self.I, np.uint64)
        self._check(lib().ps_cached_blocks(self._h, out.ctypes.data, self.I))
        return out

    def load_requests(self, req: dict):
        """Requests in flight (streaming): inst, state (0 queued FIFO / 1 decoding), L, out, rem."""
        a = [np.ascontiguousarray(req[k], dtype=d) for k, d in
             (("inst", np.uint32), ("state", np.uint32), ("L", np.uint32), ("out", np.uint32), ("rem", np.uint64))]
        n = a[0].shape[0]
        self._check(lib().ps_load_requests(self._h, n, *[x.ctypes.data if n else None for x in a]))

    def advance_window(self, window_ms: float = 20.0, prefill_tokens: int = 1000, evict: bool = True):
        p = PsAdvanceParams(float(window_ms), int(prefill_tokens), 1 if evict else 0)
        self._check(lib().ps_advance_window(self._h, ctypes.byref(p)))

    def timings(self) -> dict:
        """Device ms of the last call's kernels: probe phase, score, greedy, commit, and the probe
        phase's parts (relations, probe_scratch, probe_derived); -1 where a kernel did not run."""
        ms = np.zeros(7, np.float32)
        self._check(lib().ps_last_timings(self._h, ms.ctypes.data, 7))
        names = ("probe", "score", "greedy", "commit", "relations", "probe_scratch", "probe_derived")
        return dict(zip(names, (float(x) for x in ms)))

    def calibrate(self, batch, ctx_tokens, measured_ms, weight: float = 0.02):
        """Online calibration (ps_calibrate): pure-decode samples, in order."""
        b = np.ascontiguousarray(batch, np.int32)
        c = np.ascontiguousarray(ctx_tokens, np.int64)
        t = np.ascontiguousarray(measured_ms, np.float32)
        if not (b.shape == c.shape == t.shape):
            raise ValueError("one batch size, context and duration per sample")
        n = b.shape[0]
        self._check(lib().ps_calibrate(self._h, n, b.ctypes.data if n else None, c.ctypes.data if n else None,
                                       t.ctypes.data if n else None, float(weight)))

    def ema_factors(self) -> np.ndarray:
        out = np.zeros(16, np.float32)
        self._check(lib().ps_get_ema_factors(self._h, out.ctypes.data, 16))
        return out

    def set_model(self, model: dict):
        """Replace the performance model (ps_set_model); the EMA factors become the model's."""
        m = make_model(model)
        self._check(lib().ps_set_model(self._h, ctypes.byref(m)))
        self.selector = int(m.selector)

    def set_wait_limit(self, ns: int = 0):
        """Bound on the greedy pass's cross-block waits (ps_set_wait_limit; 0 = the 1-s default)."""
        self._check(lib().ps_set_wait_limit(self._h, int(ns)))

    def probe_stats(self) -> dict:
        """Counters of the last probe phase (see ps_last_probe_stats)."""
        v = np.zeros(16, np.uint64)
        self._check(lib().ps_last_probe_stats(self._h, v.ctypes.data, 16))
        names = ("rows_scratch", "rows_derived", "lookups_scratch", "lookups_derived", "chain_reads",
                 "pairs_derived", "greedy_fast", "greedy_full", "cyc_decide_wait", "cyc_decide_total",
                 "cyc_feed_slot_wait", "cyc_feed_summary_wait", "cyc_summary_job_wait",
                 "cyc_summary_ready_wait", "cyc_summary_eval", "cyc_probe_insert_wait")
        return dict(zip(names, (int(x) for x in v)))

    # ------------------------------------------------------------------------------------------
    @staticmethod
    def make_window(window) -> PsWindow:
        """A PsWindow over a workload.Window-like object of numpy arrays or CUDA tensors."""
        w = PsWindow()
        arrs = [(window.chain_off, np.uint64), (window.chain_hash, np.uint64),
                (window.prompt_tokens, np.uint32), (window.ttft_target, np.float32),
                (window.tpot_target, np.float32), (getattr(window, "out_tokens", None), np.uint32),
                (getattr(window, "parent", None), np.int32)]
        ptrs = [_ptr(a, d) for a, d in arrs]
        dev = {p[1] for p in ptrs if p[1] is not None}
        if len(dev) > 1:
            raise ValueError("window arrays must all be host or all be device")
        n_off = window.chain_off.numel() if _is_torch(window.chain_off) else window.chain_off.shape[0]
        w.R = int(n_off) - 1
        (w.chain_off, w.chain_hash, w.prompt_tokens, w.ttft_target, w.tpot_target, w.out_tokens,
         w.parent) = (p[0] for p in ptrs)
        w.inputs_on_device = 1 if dev == {True} else 0
        return w

    def _outputs(self, R: int, names, device_outputs: bool):
        shapes = {"hits": ((R, self.I), np.uint32), "tpot": ((R, self.I), np.float32),
                  "ttft": ((R, self.I), np.float32), "cls": ((R, self.I), np.uint8),
                  "best": ((R,), np.int32), "path": ((R,), np.uint8), "assign": ((R,), np.int32),
                  "dpath": ((R,), np.uint8), "hit_chosen": ((R,), np.uint32)}
        out = {}
        for n in names:
            shp, dt = shapes[n]
            if device_outputs:
                import torch
                tdt = {np.uint32: torch.int32, np.float32: torch.float32, np.uint8: torch.uint8,
                       np.int32: torch.int32}[dt]
                out[n] = torch.empty(shp, dtype=tdt, device=f"cuda:{self.device}")
            else:
                out[n] = np.zeros(shp, dt)
        return out

    def _scores_struct(self, o: dict, device_outputs: bool) -> PsScores:
        sc = PsScores()
        for n in ("hits", "tpot", "ttft", "cls", "best", "path"):
            setattr(sc, n, _ptr(o[n])[0] if n in o else None)
        sc.outputs_on_device = 1 if device_outputs else 0
        return sc

    def score_window(self, window, want=("hits", "tpot", "ttft", "cls", "best", "path"),
                     device_outputs: bool = False) -> dict:
        w = self.make_window(window)
        o = self._outputs(w.R, want, device_outputs)
        sc = self._scores_struct(o, device_outputs)
        self._check(lib().ps_score_window(self._h, ctypes.byref(w), ctypes.byref(sc)))
        return o

    def schedule_window(self, window, scores=(), device_outputs: bool = False) -> dict:
        """Greedy decisions {assign, path, hit_chosen}; with ``scores`` (names as score_window)
        also {"scores": {...}}: the independent scores of the window against the committed state."""
        w = self.make_window(window)
        o = self._outputs(w.R, ("assign", "dpath", "hit_chosen"), device_outputs)
        d = PsDecisions()
        d.assign, d.path, d.hit_chosen = (_ptr(o[n])[0] for n in ("assign", "dpath", "hit_chosen"))
        d.outputs_on_device = 1 if device_outputs else 0
        so = self._outputs(w.R, tuple(scores), device_outputs) if scores else {}
        sc = self._scores_struct(so, device_outputs) if scores else None
        self._check(lib().ps_schedule_window(self._h, ctypes.byref(w), ctypes.byref(d),
                                             ctypes.byref(sc) if sc is not None else None))
        res = {"assign": o["assign"], "path": o["dpath"], "hit_chosen": o["hit_chosen"]}
        if scores:
            res["scores"] = so
        return res

    def commit_window(self, last_use: int = 0):
        self._check(lib().ps_commit_window(self._h, int(last_use)))

    # -- column-block scoring (see paper_2609_33224_gb300.shard) -------------------------------
    def shard_wmin(self, window, device_outputs: bool = False):
        """ps_shard_wmin: this context's W_min over A per request (order-preserving u32 bits)."""
        w = self.make_window(window)
        if device_outputs:
            import torch
            out = torch.empty(w.R, dtype=torch.int32, device=f"cuda:{self.device}")
        else:
            out = np.zeros(w.R, np.uint32)
        self._check(lib().ps_shard_wmin(self._h, ctypes.byref(w), _ptr(out)[0], 1 if device_outputs else 0))
        return out

    def shard_pick(self, wmin_ord, id_base: int, scores=(), device_outputs: bool = False) -> dict:
        """ps_shard_pick: {key (u64), tie (u32)} per request under the pool's W_min ``wmin_ord`` (host
        u32 array, or a CUDA int32 tensor with device_outputs), plus this block's ``scores``."""
        R = wmin_ord.numel() if _is_torch(wmin_ord) else len(wmin_ord)
        if device_outputs:
            import torch
            key = torch.empty(R, dtype=torch.int64, device=f"cuda:{self.device}")
            tie = torch.empty(R, dtype=torch.int32, device=f"cuda:{self.device}")
        else:
            wmin_ord = np.ascontiguousarray(wmin_ord, dtype=np.uint32)
            key, tie = np.zeros(R, np.uint64), np.zeros(R, np.uint32)
        so = self._outputs(R, tuple(scores), device_outputs) if scores else {}
        sc = self._scores_struct(so, device_outputs) if scores else None
        self._check(lib().ps_shard_pick(self._h, _ptr(wmin_ord)[0], int(id_base), _ptr(key)[0], _ptr(tie)[0],
                                        1 if device_outputs else 0, ctypes.byref(sc) if sc is not None else None))
        res = {"key": key, "tie": tie}
        if scores:
            res["scores"] = so
        return res


def scheduler_for(workload, max_window_chain_blocks: int | None = None, device: int = 0, stream=None,
                  model: dict | None = None, load: bool = True,
                  probe_mode: int = PS_PROBE_SEARCH, track_lru: bool = False,
                  max_active_requests: int = 0, max_window_requests: int | None = None) -> Scheduler:
    """A context sized for a workload.Workload, optionally seeded with its instances."""
    win, ins = workload.window, workload.instances
    mb = max_window_chain_blocks or max(1, int(win.chain_off[-1]))
    s = Scheduler(ins.I, ins.cap_blocks, max(1, max_window_requests or win.R), mb, model or workload.model,
                  table_load_factor=workload.table_load_factor, device=device, stream=stream,
                  probe_mode=probe_mode, track_lru=track_lru, max_active_requests=max_active_requests)
    if load:
        s.load_workload_instances(ins)
    return s
