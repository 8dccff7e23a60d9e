"""The oracle reproduces its stored outputs on workload c1 and on a small
layout-branch workload with a paged prefix (regression pins; the stored
values were written by tests/golden/make_golden.py from the oracle alone)."""
import os

import numpy as np

import oracle
from paper_2607_18839_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "c1_oracle.txt")
GOLDEN_LAYOUT = os.path.join(os.path.dirname(__file__), "golden", "layout_oracle.txt")


def load_golden(path=GOLDEN):
    lse, out = {}, {}
    with open(path) as f:
        for line in f:
            if line.startswith("#"):
                continue
            t = line.split()
            if t[0] == "lse":
                lse[(int(t[1]), int(t[2]))] = float(t[3])
            else:
                out[(int(t[1]), int(t[2]), int(t[3]))] = float(t[4])
    return lse, out


def test_oracle_reproduces_stored_c1_values():
    inp = W.make_config("c1")
    o, l = oracle.branch_attn(inp)
    lse, out = load_golden()
    assert len(lse) == inp.rows * inp.H_q
    for (r, h), v in lse.items():
        assert abs(l[r, h] - v) <= 1e-12
    for (r, h, c), v in out.items():
        assert abs(o[r, h, c] - v) <= 1e-12


def test_oracle_reproduces_stored_layout_values():
    import sys
    sys.path.insert(0, os.path.join(os.path.dirname(__file__), "golden"))
    from make_golden import layout_case
    inp = layout_case()
    o, l = oracle.branch_attn(inp)
    lse, out = load_golden(GOLDEN_LAYOUT)
    assert len(lse) == inp.rows * inp.H_q
    for (r, h), v in lse.items():
        assert abs(l[r, h] - v) <= 1e-12
    for (r, h, c), v in out.items():
        assert abs(o[r, h, c] - v) <= 1e-12
