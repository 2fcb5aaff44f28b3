"""Seeded synthetic scheduling windows (inputs only; no scheduler arithmetic here).

The native generator ``gen.cpp`` draws sessions, instance caches, instance state and the window's
requests.  This module compiles it on first use, names the five workload configurations and
returns their arrays as numpy buffers that both the oracle and the CUDA library consume.

Model coefficients are the synthetic white-box fits every configuration shares: prefill
``5 + 0.02*new + 1e-6*new*ctx`` ms with ``ctx = cached + new`` (paper Eq. 6 with
alpha0=5, alpha1=0.02, alpha2=alpha3=1e-6), decode ``8 + 0.15*batch + 2e-5*kv_tokens`` ms (Eq. 7)
and ``0.004`` ms of TPOT per queued prefill token.  eta = 0.5 is the paper's default recompute
budget (Section 8.1 setup).

KV tokens held (S): config 0 uses the sum of the instance's cached session lengths, as that
configuration states.  The larger configurations cache far more session tokens than an instance's
KV capacity M_KV = 16 x cap_blocks can hold for its decode batch, so there S is also bounded by
M_KV x b / B_max: each of the b decoding requests holds at most its share of KV per decode slot.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "libws.so")
_LOCK = threading.Lock()
_LIB = None


class WsParams(ctypes.Structure):
    _fields_ = [
        ("seed", ctypes.c_uint64),
        ("num_instances", ctypes.c_uint32), ("window_requests", ctypes.c_uint32),
        ("num_sessions", ctypes.c_uint32),
        ("steps_lo", ctypes.c_uint32), ("steps_hi", ctypes.c_uint32),
        ("inc_mu", ctypes.c_double), ("inc_sigma", ctypes.c_double),
        ("ctx_min", ctypes.c_uint32), ("ctx_start_hi", ctypes.c_uint32),
        ("ctx_max", ctypes.c_uint32),
        ("sys_tokens", ctypes.c_uint32),
        ("zipf_s", ctypes.c_double),
        ("affinity", ctypes.c_double),
        ("fork_every", ctypes.c_uint32),
        ("hist_lo", ctypes.c_uint32), ("hist_hi", ctypes.c_uint32),
        ("cap_blocks", ctypes.c_uint64),
        ("fill_lo", ctypes.c_double), ("fill_hi", ctypes.c_double),
        ("b_hi", ctypes.c_uint32),
        ("q_hi", ctypes.c_uint64),
        ("b_max", ctypes.c_uint32),
        ("tpot_target_ms", ctypes.c_float), ("ttft_target_ms", ctypes.c_float),
        ("out_mu", ctypes.c_double), ("out_sigma", ctypes.c_double),
        ("out_lo", ctypes.c_uint32), ("out_hi", ctypes.c_uint32),
        ("kv_rule", ctypes.c_uint32),
    ]


def build(force: bool = False) -> str:
    """Compile the generator (plain g++, no -march flags: identical output on x86-64 and aarch64)."""
    with _LOCK:
        src = os.path.join(_HERE, "gen.cpp")
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
        lib.ws_generate.restype = ctypes.c_void_p
        lib.ws_generate.argtypes = [ctypes.POINTER(WsParams)]
        lib.ws_next_window.argtypes = [ctypes.c_void_p, ctypes.c_uint32]
        lib.ws_sizes.argtypes = [ctypes.c_void_p, ctypes.c_void_p]
        lib.ws_copy_window.argtypes = [ctypes.c_void_p] + [ctypes.c_void_p] * 7
        lib.ws_copy_instances.argtypes = [ctypes.c_void_p] + [ctypes.c_void_p] * 7
        lib.ws_copy_seed_chains.argtypes = [ctypes.c_void_p] + [ctypes.c_void_p] * 4
        lib.ws_release_seed_chains.argtypes = [ctypes.c_void_p]
        lib.ws_free.argtypes = [ctypes.c_void_p]
        lib.ws_chain_from_tokens.restype = ctypes.c_uint64
        lib.ws_chain_from_tokens.argtypes = [ctypes.c_void_p, ctypes.c_uint64, ctypes.c_void_p]
        lib.ws_initial_requests.restype = ctypes.c_uint64
        lib.ws_initial_requests.argtypes = [ctypes.c_void_p] * 6
        lib.ws_det_exp.restype = ctypes.c_double
        lib.ws_det_exp.argtypes = [ctypes.c_double]
        lib.ws_det_log.restype = ctypes.c_double
        lib.ws_det_log.argtypes = [ctypes.c_double]
        _LIB = lib
    return _LIB


def _p(a: np.ndarray) -> int:
    return a.ctypes.data


# Shared synthetic latency model (see module docstring).
MODEL_DEFAULT = dict(a0=5.0, a1=0.02, a2=1e-6, a3=1e-6, a4=0.0, a5=0.0,
                     b0=8.0, b1=0.15, b2=2e-5, g_q=0.004, eta=0.5, lout_median=556.0,
                     interference_mode=0, ttft_filter=1, seg_lo=[0], ema_factor=[1.0])

_COMMON = dict(steps_lo=8, steps_hi=40, inc_mu=7.5, inc_sigma=0.8, affinity=0.8, fork_every=0,
               hist_lo=0, hist_hi=40, fill_lo=1.0, fill_hi=1.0, out_mu=6.1, out_sigma=0.6,
               out_lo=16, out_hi=4096, kv_rule=1)

# The five workloads.  ``table_load_factor`` sizes the instance hash tables (slots = cap / lf).
CONFIGS = {
    # tiny window: 8 instances x 64 requests, 4 sessions, prompts 1K-8K tokens
    0: dict(_COMMON, seed=0, num_instances=8, window_requests=64, num_sessions=4, steps_lo=3,
            steps_hi=8, inc_mu=7.0, inc_sigma=0.5, ctx_min=1024, ctx_start_hi=4096, ctx_max=8192,
            sys_tokens=0, zipf_s=0.0, hist_hi=8, cap_blocks=4096, fill_lo=0.5, fill_hi=1.0, kv_rule=0,
            b_hi=32, q_hi=8192, b_max=64, tpot_target_ms=50.0, ttft_target_ms=2000.0,
            table_load_factor=0.5),
    # eval-scale window: 64 instances x 4096 requests, 512 sessions, contexts 8K-128K
    1: dict(_COMMON, seed=1, num_instances=64, window_requests=4096, num_sessions=512,
            ctx_min=8192, ctx_start_hi=65536, ctx_max=131072, sys_tokens=4096, zipf_s=0.0,
            cap_blocks=65536, b_hi=64, q_hi=8192, b_max=128, tpot_target_ms=50.0,
            ttft_target_ms=2000.0, table_load_factor=0.5),
    # production-scale window: 1024 instances x 16384 requests, 8192 Zipf(1.1) sessions
    2: dict(_COMMON, seed=2, num_instances=1024, window_requests=16384, num_sessions=8192,
            ctx_min=4096, ctx_start_hi=65536, ctx_max=131072, sys_tokens=4096, zipf_s=1.1,
            cap_blocks=200000, b_hi=128, q_hi=32768, b_max=256, tpot_target_ms=50.0,
            ttft_target_ms=3000.0, table_load_factor=0.9),
    # long-context stress: 256 instances x 2048 requests, prefixes 128K-1M, 32K shared prompt
    3: dict(_COMMON, seed=3, num_instances=256, window_requests=2048, num_sessions=4096,
            ctx_min=131072, ctx_start_hi=524288, ctx_max=1048576, sys_tokens=32768, zipf_s=1.1,
            fork_every=10, hist_hi=20, cap_blocks=1 << 20, b_hi=128, q_hi=32768, b_max=256,
            tpot_target_ms=30.0, ttft_target_ms=3000.0, table_load_factor=0.5),
    # streaming: 1024 instances, 1000 windows of 1000 requests, state carried across windows.
    # A commit merges a window's blocks before eviction runs; the capacity guard bounds an
    # instance's admitted blocks per window by its KV capacity (= cap blocks), so tables get
    # 2 x cap slots.
    4: dict(_COMMON, seed=4, num_instances=1024, window_requests=1000, num_sessions=8192,
            ctx_min=4096, ctx_start_hi=65536, ctx_max=131072, sys_tokens=4096, zipf_s=1.1,
            cap_blocks=200000, b_hi=128, q_hi=32768, b_max=256, tpot_target_ms=50.0,
            ttft_target_ms=3000.0, table_load_factor=0.5),
}


@dataclass
class Window:
    """One window of requests in arrival order (chains as CSR)."""
    chain_off: np.ndarray      # u64[R+1]
    chain_hash: np.ndarray     # u64[sum nb]
    prompt_tokens: np.ndarray  # u32[R]
    ttft_target: np.ndarray    # f32[R] (ms)
    tpot_target: np.ndarray    # f32[R] (ms)
    session: np.ndarray        # u32[R]
    out_tokens: np.ndarray     # u32[R] (streaming windows only)

    @property
    def R(self) -> int:
        return int(self.prompt_tokens.shape[0])


@dataclass
class Instances:
    """Instance state (SoA) and seed cache contents (chains as CSR with a parent hash each)."""
    b: np.ndarray        # i32[I] decoding requests
    qr: np.ndarray       # i32[I] queued requests
    q: np.ndarray        # i64[I] queued prefill tokens
    S: np.ndarray        # i64[I] KV tokens held
    M_KV: np.ndarray     # i64[I] KV token capacity
    B_max: np.ndarray    # i32[I] decode-slot limit
    cap_blocks: np.ndarray   # u64[I] cache capacity (blocks)
    chain_inst: np.ndarray   # u32[nc]
    chain_off: np.ndarray    # u64[nc+1]
    chain_hash: np.ndarray   # u64[...]
    chain_parent: np.ndarray  # u64[nc] (0 = root)

    @property
    def I(self) -> int:
        return int(self.b.shape[0])


@dataclass
class TreeWindow:
    """A window in the shared-prefix form: request r's chain is request parent[r]'s whole chain
    followed by its own blocks chain_hash[chain_off[r]:chain_off[r+1]] (parent -1: the whole chain)."""
    chain_off: np.ndarray      # u64[R+1] own blocks
    chain_hash: np.ndarray     # u64[sum own]
    prompt_tokens: np.ndarray  # u32[R]
    ttft_target: np.ndarray    # f32[R]
    tpot_target: np.ndarray    # f32[R]
    session: np.ndarray        # u32[R]
    out_tokens: np.ndarray     # u32[R]
    parent: np.ndarray         # i32[R]

    @property
    def R(self) -> int:
        return int(self.prompt_tokens.shape[0])


def tree_window(win: Window) -> TreeWindow:
    """The shared-prefix form of a window: each request's parent is the latest earlier request of its
    session whose chain is a prefix of its own (chained block hashes: equal hashes at the parent's
    last position mean equal prefixes), and only the blocks after the parent's chain are kept."""
    off = win.chain_off.astype(np.int64)
    R = win.R
    parent = np.full(R, -1, np.int32)
    by_session: dict = {}
    for r in range(R):
        a, b = int(off[r]), int(off[r + 1])
        for p in reversed(by_session.get(int(win.session[r]), [])):
            pa, pb = int(off[p]), int(off[p + 1])
            n = pb - pa
            if 0 < n <= b - a and win.chain_hash[pb - 1] == win.chain_hash[a + n - 1]:
                parent[r] = p
                break
        by_session.setdefault(int(win.session[r]), []).append(r)
    keep = np.ones(int(off[-1]), bool)
    own = np.zeros(R + 1, np.uint64)
    for r in range(R):
        p = int(parent[r])
        n = int(off[p + 1] - off[p]) if p >= 0 else 0
        keep[int(off[r]):int(off[r]) + n] = False
        own[r + 1] = own[r] + np.uint64(int(off[r + 1] - off[r]) - n)
    return TreeWindow(chain_off=own, chain_hash=win.chain_hash[keep].astype(np.uint64),
                      prompt_tokens=win.prompt_tokens, ttft_target=win.ttft_target, tpot_target=win.tpot_target,
                      session=win.session, out_tokens=win.out_tokens, parent=parent)


def column_block(ins: Instances, lo: int, hi: int) -> Instances:
    """Instances lo .. hi - 1 of a pool as a pool of their own (ids renumbered from 0): the seed
    chains cached on them and their state."""
    sel = np.nonzero((ins.chain_inst >= lo) & (ins.chain_inst < hi))[0]
    lens = np.diff(ins.chain_off)[sel].astype(np.uint64)
    off = np.zeros(sel.shape[0] + 1, np.uint64)
    off[1:] = np.cumsum(lens)
    hashes = [ins.chain_hash[int(ins.chain_off[c]):int(ins.chain_off[c + 1])] for c in sel]
    return Instances(b=ins.b[lo:hi].copy(), qr=ins.qr[lo:hi].copy(), q=ins.q[lo:hi].copy(),
                     S=ins.S[lo:hi].copy(), M_KV=ins.M_KV[lo:hi].copy(), B_max=ins.B_max[lo:hi].copy(),
                     cap_blocks=ins.cap_blocks[lo:hi].copy(),
                     chain_inst=(ins.chain_inst[sel] - lo).astype(np.uint32), chain_off=off,
                     chain_hash=(np.concatenate(hashes) if hashes else np.zeros(0, np.uint64)).astype(np.uint64),
                     chain_parent=ins.chain_parent[sel].copy())


@dataclass
class Workload:
    config: int
    params: dict
    table_load_factor: float
    window: Window
    instances: Instances
    model: dict = field(default_factory=lambda: dict(MODEL_DEFAULT))
    _handle: int | None = None

    def next_window(self, R: int | None = None) -> Window:
        """Streaming: draw the next window (sessions continue where the last window left them)."""
        lib = _lib()
        lib.ws_next_window(self._handle, int(self.params["window_requests"] if R is None else R))
        self.window = _copy_window(self._handle)
        return self.window

    def initial_requests(self) -> dict:
        """Requests in flight at the start of a stream (see ws_initial_requests in gen.cpp):
        inst, state (0 queued in FIFO order, 1 decoding), L, out, rem."""
        lib = _lib()
        n = int(lib.ws_initial_requests(self._handle, None, None, None, None, None))
        r = dict(inst=np.zeros(n, np.uint32), state=np.zeros(n, np.uint32), L=np.zeros(n, np.uint32),
                 out=np.zeros(n, np.uint32), rem=np.zeros(n, np.uint64))
        if n:
            lib.ws_initial_requests(self._handle, _p(r["inst"]), _p(r["state"]), _p(r["L"]), _p(r["out"]),
                                    _p(r["rem"]))
        return r

    def close(self):
        if self._handle is not None:
            _lib().ws_free(self._handle)
            self._handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def _sizes(h) -> np.ndarray:
    out = np.zeros(5, dtype=np.uint64)
    _lib().ws_sizes(h, _p(out))
    return out


def _copy_window(h) -> Window:
    _, R, nblk, _, _ = (int(x) for x in _sizes(h))
    w = Window(chain_off=np.zeros(R + 1, np.uint64), chain_hash=np.zeros(nblk, np.uint64),
               prompt_tokens=np.zeros(R, np.uint32), ttft_target=np.zeros(R, np.float32),
               tpot_target=np.zeros(R, np.float32), session=np.zeros(R, np.uint32),
               out_tokens=np.zeros(R, np.uint32))
    _lib().ws_copy_window(h, _p(w.chain_off), _p(w.chain_hash), _p(w.prompt_tokens),
                          _p(w.ttft_target), _p(w.tpot_target), _p(w.session), _p(w.out_tokens))
    return w


def generate(config: int | dict, **overrides) -> Workload:
    """Generate a workload: a config index (0-4) or a full parameter dict, with overrides."""
    if isinstance(config, dict):
        params = dict(config)
        cid = -1
    else:
        cid = int(config)
        params = dict(CONFIGS[cid])
    params.update(overrides)
    lf = float(params.pop("table_load_factor", 0.5))
    wp = WsParams(**{k: params[k] for k, _ in WsParams._fields_})
    lib = _lib()
    h = lib.ws_generate(ctypes.byref(wp))
    if not h:
        raise ValueError("invalid workload parameters")
    I, R, nblk, nc, nseed = (int(x) for x in _sizes(h))
    window = _copy_window(h)
    inst = Instances(b=np.zeros(I, np.int32), qr=np.zeros(I, np.int32), q=np.zeros(I, np.int64),
                     S=np.zeros(I, np.int64), M_KV=np.zeros(I, np.int64),
                     B_max=np.zeros(I, np.int32), cap_blocks=np.zeros(I, np.uint64),
                     chain_inst=np.zeros(nc, np.uint32), chain_off=np.zeros(nc + 1, np.uint64),
                     chain_hash=np.zeros(nseed, np.uint64), chain_parent=np.zeros(nc, np.uint64))
    lib.ws_copy_instances(h, _p(inst.b), _p(inst.qr), _p(inst.q), _p(inst.S), _p(inst.M_KV),
                          _p(inst.B_max), _p(inst.cap_blocks))
    lib.ws_copy_seed_chains(h, _p(inst.chain_inst), _p(inst.chain_off), _p(inst.chain_hash),
                            _p(inst.chain_parent))
    lib.ws_release_seed_chains(h)
    params["table_load_factor"] = lf
    return Workload(config=cid, params=params, table_load_factor=lf, window=window,
                    instances=inst, _handle=h)


def chain_from_tokens(tokens) -> np.ndarray:
    """Block-hash chain (full 16-token blocks) of an explicit token list."""
    t = np.ascontiguousarray(np.asarray(tokens, dtype=np.uint32))
    out = np.zeros(max(1, t.shape[0] // 16), np.uint64)
    n = _lib().ws_chain_from_tokens(_p(t), t.shape[0], _p(out))
    return out[:n]


def det_exp(x: float) -> float:
    return _lib().ws_det_exp(float(x))


def det_log(x: float) -> float:
    return _lib().ws_det_log(float(x))
