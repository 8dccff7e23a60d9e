"""Write the stored oracle outputs under tests/golden/.

Calls only the oracle (and the seeded input generator): no value here comes
from the CUDA library.  Re-run after a change to the oracle's arithmetic,
and name the passage of the paper that justifies the change in the commit.

    python tests/golden/make_golden.py
"""
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import oracle  # noqa: E402
from paper_2607_18839_gb300 import workloads as W  # noqa: E402


def main():
    inp = W.make_config("c1")
    out, lse = oracle.branch_attn(inp)
    path = os.path.join(HERE, "c1_oracle.txt")
    with open(path, "w") as f:
        f.write("# fp64 oracle on workload c1 (seed 1001): one page, prefix 256, 4 branches\n")
        f.write("# with private histories 8/16/24/32, m=1, H_q=8, H_kv=2, D=64.\n")
        f.write("# Written by tests/golden/make_golden.py from oracle/ only.\n")
        f.write("# lines: 'lse row head value' and 'out row head c value' (heads 0 and 7)\n")
        for r in range(inp.rows):
            for h in range(inp.H_q):
                f.write(f"lse {r} {h} {lse[r, h]:.17g}\n")
        for r in range(inp.rows):
            for h in (0, inp.H_q - 1):
                for c in range(inp.D):
                    f.write(f"out {r} {h} {c} {out[r, h, c]:.17g}\n")
    print("wrote", path)


if __name__ == "__main__":
    main()
