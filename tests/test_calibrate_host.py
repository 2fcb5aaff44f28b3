"""The library's online-calibration update (paper_2609_33224_gb300/csrc/calibrate.h, the host code
behind ps_calibrate) against the oracle's, bit for bit, on random pure-decode samples that reach
both clips and every segment.  The header is plain C++; here it is compiled into a small harness
with the library's host flags (no floating-point contraction)."""
import os
import subprocess

import numpy as np
import pytest

import workload as W
from oracle import Oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2609_33224_gb300", "csrc")

HARNESS = r"""
#include <cstdio>
#include <vector>
#include "calibrate.h"
int main() {
  float b0, b1, b2, w; int nseg; unsigned long long n;
  if (std::fread(&b0, 4, 1, stdin) != 1 || std::fread(&b1, 4, 1, stdin) != 1 || std::fread(&b2, 4, 1, stdin) != 1 ||
      std::fread(&w, 4, 1, stdin) != 1 || std::fread(&nseg, 4, 1, stdin) != 1 || std::fread(&n, 8, 1, stdin) != 1)
    return 1;
  std::vector<int32_t> lo(nseg), batch(n);
  std::vector<float> f(nseg), t(n);
  std::vector<int64_t> ctx(n);
  if (std::fread(lo.data(), 4, nseg, stdin) != (size_t)nseg || std::fread(f.data(), 4, nseg, stdin) != (size_t)nseg ||
      std::fread(batch.data(), 4, n, stdin) != n || std::fread(ctx.data(), 8, n, stdin) != n ||
      std::fread(t.data(), 4, n, stdin) != n)
    return 1;
  pscal::ema_update(b0, b1, b2, nseg, lo.data(), f.data(), n, batch.data(), ctx.data(), t.data(), w);
  std::fwrite(f.data(), 4, nseg, stdout);
  return 0;
}
"""


@pytest.fixture(scope="module")
def harness(tmp_path_factory):
    d = tmp_path_factory.mktemp("calib")
    src, exe = d / "h.cpp", d / "h"
    src.write_text(HARNESS)
    subprocess.run(["g++", "-std=c++17", "-O2", "-ffp-contract=off", "-I", CSRC, str(src), "-o", str(exe)],
                   check=True)
    return str(exe)


def _run(exe, m, lo, f0, batch, ctx, t, w):
    blob = (np.array([m["b0"], m["b1"], m["b2"], w], np.float32).tobytes() +
            np.array([len(lo)], np.int32).tobytes() + np.array([len(batch)], np.uint64).tobytes() +
            np.asarray(lo, np.int32).tobytes() + np.asarray(f0, np.float32).tobytes() +
            np.asarray(batch, np.int32).tobytes() + np.asarray(ctx, np.int64).tobytes() +
            np.asarray(t, np.float32).tobytes())
    out = subprocess.run([exe], input=blob, capture_output=True, check=True).stdout
    return np.frombuffer(out, np.float32)


@pytest.mark.parametrize("seed,weight", [(0, 0.02), (1, 0.02), (2, 0.3), (3, 1.0)])
def test_library_update_matches_oracle_bit_for_bit(harness, seed, weight):
    rng = np.random.default_rng(seed)
    lo = [0, 9, 17, 33, 65, 129]
    n = 5000
    batch = rng.integers(0, 300, n)
    ctx = rng.integers(0, 2_000_000, n)
    base = (8.0 + 0.15 * batch) + 2e-5 * ctx
    t = (base * rng.uniform(0.2, 3.0, n)).astype(np.float32)  # ratios below 0.5 and above 2 included
    model = dict(W.MODEL_DEFAULT, seg_lo=lo, ema_factor=[1.0] * len(lo))
    o = Oracle(1, model)
    o.calibrate(batch, ctx, t, weight=weight)
    want = o.ema_factors()
    got = _run(harness, model, lo, [1.0] * len(lo), batch, ctx, t, weight)
    assert got.view(np.uint32).tolist() == want.view(np.uint32).tolist()
    assert np.all(got >= 1.0) and np.all(got <= 2.0)
