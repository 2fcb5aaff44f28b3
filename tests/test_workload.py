"""The seeded generator: deterministic, well-formed CSR, prefix structure of agentic sessions."""
import numpy as np

import workload as W


def test_deterministic_and_seeded():
    a, b = W.generate(0), W.generate(0)
    assert np.array_equal(a.window.chain_hash, b.window.chain_hash)
    assert np.array_equal(a.instances.chain_hash, b.instances.chain_hash)
    assert np.array_equal(a.instances.q, b.instances.q)
    c = W.generate(0, seed=99)
    assert not np.array_equal(a.window.chain_hash[:100], c.window.chain_hash[:100])


def test_window_shapes_and_block_counts():
    wl = W.generate(0)
    win = wl.window
    nb = np.diff(win.chain_off).astype(np.int64)
    assert win.R == 64 and win.chain_off[0] == 0
    assert np.array_equal(nb, win.prompt_tokens.astype(np.int64) // 16)
    assert np.all(win.prompt_tokens >= 1024) and np.all(win.prompt_tokens <= 8192)
    assert np.all(win.chain_hash != 0)


def test_session_steps_extend_prefixes():
    """Consecutive requests of one session share the earlier prompt as a chain prefix."""
    wl = W.generate(0)
    win = wl.window
    last = {}
    extended = 0
    for r in range(win.R):
        s = int(win.session[r])
        ch = win.chain_hash[win.chain_off[r]:win.chain_off[r + 1]]
        if s in last and last[s].shape[0] <= ch.shape[0] and np.array_equal(ch[:last[s].shape[0]], last[s]):
            extended += 1
        last[s] = ch
    assert extended >= win.R // 2


def test_instance_fill_and_state_ranges():
    wl = W.generate(0)
    ins = wl.instances
    per = np.bincount(ins.chain_inst, weights=np.diff(ins.chain_off).astype(np.float64), minlength=ins.I)
    assert np.all(per <= 4096) and np.all(per >= 2048)
    assert np.all((ins.b >= 0) & (ins.b <= 32)) and np.all((ins.q >= 0) & (ins.q <= 8192))
    assert np.array_equal(ins.qr, (ins.q + 4095) // 4096)
    assert np.all(ins.S <= ins.M_KV) and np.all(ins.M_KV == 16 * 4096)


def test_chain_from_tokens_matches_generator_chaining():
    """The block hash of block k covers tokens [0, 16(k+1)): equal prefixes, equal hashes."""
    t = np.arange(100, dtype=np.uint32)
    a = W.chain_from_tokens(t)
    b = W.chain_from_tokens(np.concatenate([t[:40], t[40:] + 1]))
    assert a.shape[0] == 6 and b.shape[0] == 6
    assert np.array_equal(a[:2], b[:2]) and not np.any(a[2:] == b[2:])
    assert W.chain_from_tokens(t[:15]).shape[0] == 0


def test_deterministic_series_match_libm_closely():
    import math
    for x in (-5.0, -0.3, 0.0, 1.0, 7.5, 11.9):
        assert abs(W.det_exp(x) - math.exp(x)) <= 1e-13 * math.exp(x)
    for x in (0.5, 1.0, 3.0, 8192.0, 1e6):
        assert abs(W.det_log(x) - math.log(x)) <= 1e-14 * max(1.0, abs(math.log(x)))
