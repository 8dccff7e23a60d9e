"""The benchmark's algorithmic work per step (the numerator of its roofline)
against counts made independently of its closed forms: FLOPs as 4 D per
visible (query row, key) pair, the pairs counted key by key from each row's
visibility (Sec. 3.3: the page's prefix up to the branch's fork position,
then the branch's own keys up to the row's causal bound), and the bytes of
the prefix, Q and output from the sizes of the input arrays."""
import importlib.util
import os

import numpy as np
import pytest

from paper_2607_18839_gb300 import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def visible_pairs(inp):
    """(query row, key) pairs one query head attends to, summed over rows."""
    n = 0
    for d in range(inp.n_docs):
        P_d = int(inp.prefix_cu[d + 1] - inp.prefix_cu[d])
        for b in range(int(inp.branch_cu[d]), int(inp.branch_cu[d + 1])):
            p_b = P_d if inp.branch_prefix_len is None else min(P_d, int(inp.branch_prefix_len[b]))
            L_b = int(inp.branch_len[b])
            for i in range(inp.m):
                n += sum(1 for j in range(P_d) if j < p_b)
                n += sum(1 for j in range(L_b) if j <= L_b - inp.m + i)
    return n


CASES = {
    "c1": lambda: W.make_config("c1"),
    "c2": lambda: W.make_config("c2"),
    "fork_lengths": lambda: W.build_inputs([500, 200], [4, 3], [10, 20, 30, 40, 0, 1, 2], 3, 8, 4,
                                           64, seed=32,
                                           branch_prefix_len=[500, 0, 1, 250, 200, 63, 64]),
    "short_histories": lambda: W.build_inputs([40, 0], [3, 2], [0, 1, 2, 0, 5], 4, 4, 2, 64,
                                              seed=5),
}


@pytest.mark.parametrize("name", list(CASES))
def test_attention_flops_are_four_d_per_visible_pair(bench, name):
    inp = CASES[name]()
    per, step = bench.algorithmic_work(inp)
    want = 4.0 * inp.D * inp.H_q * visible_pairs(inp)
    assert per["branch_attn_tc"]["flops"] == want
    assert per["prefix_stage"]["flops"] + per["suffix_merge"]["flops"] == want
    assert step["flops"] == want


@pytest.mark.parametrize("name", list(CASES))
def test_attention_bytes_follow_the_arrays(bench, name):
    inp = CASES[name]()
    per, _ = bench.algorithmic_work(inp)
    # prefix K and V: per page, the keys some branch of it sees, read once
    seen = 0
    for d in range(inp.n_docs):
        P_d = int(inp.prefix_cu[d + 1] - inp.prefix_cu[d])
        lens = [P_d if inp.branch_prefix_len is None else min(P_d, int(inp.branch_prefix_len[b]))
                for b in range(int(inp.branch_cu[d]), int(inp.branch_cu[d + 1]))]
        seen += max(lens, default=0)
    row_bytes = inp.prefix_k.nbytes // max(1, inp.prefix_k.shape[0])  # H_kv x D bf16
    prefix = 2 * seen * row_bytes
    private = 2 * int(inp.branch_len.sum()) * row_bytes
    q = inp.q.nbytes
    out = inp.q.nbytes + inp.B * inp.m * inp.H_q * 4  # bf16 out + fp32 lse
    pages = int(sum(-(-int(x) // W.PAGE) for x in inp.branch_len))
    tables = 4 * pages + 4 * inp.B + 2 * 4 * (inp.n_docs + 1)
    assert per["branch_attn_tc"]["bytes"] == prefix + private + q + tables + out


def test_c4_work_matches_the_pair_count(bench):
    # the headline workload, counted the slow way once
    inp = W.make_config("c4")
    per, _ = bench.algorithmic_work(inp)
    assert per["branch_attn_tc"]["flops"] == 4.0 * inp.D * inp.H_q * visible_pairs(inp)
