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


def layout_case():
    """Two pages with their layout branches and content branches, the prefix
    paged and shared with the layout branches (paged prefix, fork limits)."""
    return W.build_layout_inputs([37, 64], [20, 0], [2, 1], [5, 17, 3], 3, 4, 2, 64, seed=3)


def write(inp, path, header):
    out, lse = oracle.branch_attn(inp)
    with open(path, "w") as f:
        for line in header:
            f.write(f"# {line}\n")
        f.write("# Written by tests/golden/make_golden.py from oracle/ only.\n")
        f.write(f"# lines: 'lse row head value' and 'out row head c value' (heads 0 and {inp.H_q - 1})\n")
        for r in range(inp.rows):
            for h in range(inp.H_q):
                f.write(f"lse {r} {h} {lse[r, h]:.17g}\n")
        for r in range(inp.rows):
            for h in (0, inp.H_q - 1):
                for c in range(inp.D):
                    f.write(f"out {r} {h} {c} {out[r, h, c]:.17g}\n")
    print("wrote", path)


def main():
    write(W.make_config("c1"), os.path.join(HERE, "c1_oracle.txt"),
          ["fp64 oracle on workload c1 (seed 1001): one page, prefix 256, 4 branches",
           "with private histories 8/16/24/32, m=1, H_q=8, H_kv=2, D=64."])
    write(layout_case(), os.path.join(HERE, "layout_oracle.txt"),
          ["fp64 oracle on a small layout-branch workload (seed 3): pages with vision 37 / 64",
           "and layout 20 / 0 tokens, 2 / 1 content branches, m=3, H_q=4, H_kv=2, D=64; the",
           "prefix is paged and shared with each page's layout branch."])


if __name__ == "__main__":
    main()
