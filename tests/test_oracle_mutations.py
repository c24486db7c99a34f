"""Planted mistakes in the oracle must be caught by the pins (CPU only).

Each case edits one spot of a copy of ``oracle/parason_oracle.c`` -- a dropped
term, a wrong sign or index, a swapped operand -- builds it, and runs every
pin in tests/oracle_pins.py against it.  At least one pin has to fail; the
real oracle passes them all (tests/test_oracle_pins.py).
"""
import os
import subprocess
import sys

import pytest

from oracle import build as obuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

# Runs every pin against one oracle build in a child process; prints the names
# of the pins that failed.  A mutant that corrupts memory and dies is caught too.
_RUNNER = """
import sys
sys.path.insert(0, sys.argv[1])
import oracle
from tests import oracle_pins as P
mutant = oracle.Oracle(sys.argv[2])
failed = []
for check in P.ALL_CHECKS:
    try:
        check(mutant)
    except Exception as exc:
        failed.append(check.__name__)
print("FAILED:" + ",".join(failed))
"""

MUTATIONS = {
    "page_index_mod": ("t / page_size]", "t % page_size]"),
    "gqa_head_mod": ("const int32_t kvh = h / group;", "const int32_t kvh = h % num_kv_heads;"),
    "dropped_scale": ("const double s = scale * dot;", "const double s = dot;"),
    "exp_sign": ("exp(scores[pos++] - m)", "exp(m - scores[pos++])"),
    "lse_drops_max": ("*lse_out = m + log(l);", "*lse_out = log(l);"),
    "unnormalised": ("o[dd] = acc[dd] / l;", "o[dd] = acc[dd];"),
    "drops_root_node": ("for (int i = 0; i < plen; ++i)\n                total += node_len[path[i]];",
                        "for (int i = 1; i < plen; ++i)\n                total += node_len[path[i]];"),
    "k_for_v": ("load_elem(v_pages, row + dd, kv_code, vs)", "load_elem(k_pages, row + dd, kv_code, vs)"),
    "e4m3_bias": ("ldexp(1.0 + (double)mant / 8.0, expo - 7)", "ldexp(1.0 + (double)mant / 8.0, expo - 8)"),
    "e4m3_subnormal": ("ldexp((double)mant / 8.0, 1 - 7)", "ldexp((double)mant / 8.0, -7)"),
    "fp8_scale_dropped": ("(double)k_scale[kvh] : 1.0", "1.0 : 1.0"),
    "merge_weight": ("wb * o_b[r * head_dim + dd]", "wa * o_b[r * head_dim + dd]"),
    "merge_lse_drops_max": ("lse_out[r] = mx + log(wa + wb);", "lse_out[r] = log(wa + wb);"),
    "row_stride_heads": ("((page * num_kv_heads + kvh) * page_size", "((page * num_q_heads + kvh) * page_size"),
    "slot_offset": ("+ t % page_size) * head_dim;", "+ t % page_size + 1) * head_dim;"),
}


@pytest.fixture(scope="module")
def source():
    with open(obuild.SRC) as f:
        return f.read()


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_mistake_is_caught(name, source, tmp_path):
    old, new = MUTATIONS[name]
    n = source.count(old)
    assert n >= 1, f"mutation site for {name} not found in the oracle source"
    lib = obuild.build_variant(source.replace(old, new), str(tmp_path), f"oracle_{name}")
    res = subprocess.run([sys.executable, "-c", _RUNNER, ROOT, lib], capture_output=True,
                         text=True, timeout=600, env={**os.environ, "OMP_NUM_THREADS": "2"})
    if res.returncode != 0:
        return          # the mutant crashed the checks: caught
    line = [ln for ln in res.stdout.splitlines() if ln.startswith("FAILED:")][-1]
    caught = [c for c in line[len("FAILED:"):].split(",") if c]
    assert caught, f"no pin caught the planted mistake {name}"


def test_unmodified_source_passes_runner(source, tmp_path):
    """Control: the same child-process runner reports no failure for the real source."""
    lib = obuild.build_variant(source, str(tmp_path), "oracle_control")
    res = subprocess.run([sys.executable, "-c", _RUNNER, ROOT, lib], capture_output=True,
                         text=True, timeout=600, env={**os.environ, "OMP_NUM_THREADS": "2"})
    assert res.returncode == 0, res.stderr[-2000:]
    assert res.stdout.strip().splitlines()[-1] == "FAILED:"
