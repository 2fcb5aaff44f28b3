"""The C-ABI library builds, loads without a GPU, exports every entry point declared in
include/*.h, and the binding's struct layouts match the C compiler's (no compute calls here)."""
import ctypes
import glob
import os
import re
import subprocess

import pytest

import paper_2609_33224_gb300 as P

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    P.build()
    return P.lib()


def _declared():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        src = open(h).read()
        names |= set(re.findall(r"^PS_API\s+[\w\s\*]+?\b(ps_\w+)\s*\(", src, flags=re.M))
    return names


def test_every_declared_symbol_is_exported(lib):
    names = _declared()
    assert len(names) >= 14
    out = subprocess.run(["nm", "-D", "--defined-only", P._LIB_PATH], capture_output=True, text=True,
                         check=True).stdout
    exported = set(re.findall(r"\bT (ps_\w+)$", out, flags=re.M))
    assert names <= exported, names - exported
    for n in names:
        assert hasattr(lib, n)
    assert set(P.ABI_FUNCTIONS) == names


def test_struct_layouts_match_c(tmp_path):
    src = tmp_path / "layout.c"
    src.write_text("""
#include <stdio.h>
#include <stddef.h>
#include "packserve.h"
#define P(T) printf(#T " %zu\\n", sizeof(T));
#define O(T, f) printf(#T "." #f " %zu\\n", offsetof(T, f));
int main(void) {
  P(ps_model) P(ps_config) P(ps_instance_state) P(ps_window) P(ps_scores) P(ps_decisions)
  P(ps_table_desc) P(ps_state_arrays)
  O(ps_config, model) O(ps_config, table_load_factor) O(ps_config, cap_blocks)
  O(ps_model, seg_lo) O(ps_model, ema_factor) O(ps_instance_state, B_max)
  O(ps_window, inputs_on_device) O(ps_scores, outputs_on_device) O(ps_decisions, outputs_on_device)
  O(ps_model, cache_filter_off) O(ps_model, selector)
  return 0;
}
""")
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-std=c99", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)], check=True)
    got = dict(line.rsplit(" ", 1) for line in subprocess.run([str(exe)], capture_output=True, text=True,
                                                               check=True).stdout.split("\n") if line)
    ct = {"ps_model": P.PsModel, "ps_config": P.PsConfig, "ps_instance_state": P.PsInstanceState,
          "ps_window": P.PsWindow, "ps_scores": P.PsScores, "ps_decisions": P.PsDecisions,
          "ps_table_desc": P.PsTableDesc, "ps_state_arrays": P.PsStateArrays}
    for k, v in got.items():
        if "." in k:
            t, f = k.split(".")
            assert getattr(ct[t], f).offset == int(v), k
        else:
            assert ctypes.sizeof(ct[k]) == int(v), k


def test_binding_fails_loudly_without_library(monkeypatch, tmp_path):
    monkeypatch.setattr(P, "_lib", None)
    monkeypatch.setattr(P, "_LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="build the CUDA library"):
        P.lib()


def test_create_without_gpu_reports_an_error(lib):
    """No GPU here: ps_create must fail with a status, never crash or fall back to the CPU."""
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    with pytest.raises(P.PSError):
        P.Scheduler(2, [16, 16], 4, 64, dict(__import__("workload").MODEL_DEFAULT))


def test_graft_entry_build_runs_on_cpu():
    import __graft_entry__ as g
    g.build()
    assert os.path.exists(P._LIB_PATH)


def test_every_declared_call_names_its_passage():
    """Each exported call's comment block (the text between the previous declaration and this one)
    names the passage of the paper that defines the operation (a section, equation, algorithm or
    table), or says that the paper has no counterpart."""
    cite = re.compile(r"Section \d|Eq\. ?\d|Algorithm \d|Table \d|no counterpart")
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        src = open(h).read()
        prev = 0
        for mt in re.finditer(r"^PS_API\s+[\w\s\*]+?\b(ps_\w+)\s*\([^;]*;", src, flags=re.M | re.S):
            block = src[prev:mt.start()]
            assert cite.search(block), f"{mt.group(1)}: its comment names no section, equation, algorithm or table"
            prev = mt.end()


def test_policy_switches_default_to_algorithm_1():
    """A zero-initialised ps_model's policy fields select Algorithm 1: KVC-first filter and SLO
    admission on, the LMetric fallback, the D-C-Q order; the binding's tables name Table 3 / Table 4."""
    m = P.PsModel()
    assert (m.cache_filter_off, m.slo_filter_off, m.fallback_dcq, m.selector) == (0, 0, 0, 0)
    assert P.SELECTORS["D-C-Q"] == 0 and sorted(P.SELECTORS.values()) == list(range(6))
    assert P.ABLATIONS["F"] == dict(cache_filter_off=0, slo_filter_off=0, fallback_dcq=0)
    g = P.make_model(dict(__import__("workload").MODEL_DEFAULT, **P.ABLATIONS["G"], selector=5))
    assert (g.cache_filter_off, g.slo_filter_off, g.fallback_dcq, g.selector) == (1, 1, 1, 5)
