"""The layout branch as a second workload (Sec. 3.3, Algorithm 1): each
page's layout branch decodes in the same step as the content branches forked
from it, encoded as a branch whose fork prefix is the page-aligned vision
part and whose private pages are the shared prefix's own pages (no copy).

CPU pins: the oracle's layout-branch rows equal plain causal attention over
the page's whole sequence (vision, layout tokens, drafts), written with a
library softmax; the whole workload matches the explicit-mask brute force.
GPU: parity with the oracle, element by element on small cases and on
sampled branches (every layout branch among them) at full size.
"""
import numpy as np
import pytest
from scipy.special import logsumexp, softmax

import oracle
from paper_2607_18839_gb300 import workloads as W
from test_oracle_pins import brute_force, f64

OUT_TOL = 1e-2
LSE_TOL = 1e-3


def small_cases():
    # vision lengths on and off page boundaries, no layout tokens yet, a page
    # with no content branch, m = 1 and m = 8
    yield W.build_layout_inputs([37, 64, 16], [20, 0, 45], [2, 3, 0], [5, 17, 1, 40, 9], 3, 4,
                                2, 64, seed=3)
    yield W.build_layout_inputs([100], [7], [4], [0, 3, 16, 60], 1, 8, 2, 128, seed=4)
    yield W.build_layout_inputs([15, 200], [1, 33], [1, 2], [2, 2, 2], 8, 6, 3, 64, seed=5,
                                extra_pages=4)


def causal_sequence_rows(inp, d):
    """Direct causal attention of page d's layout-branch queries over the
    page's own sequence: query i sees tokens [0, P_d + i]."""
    G = inp.H_q // inp.H_kv
    scale = inp.scale or 1.0 / np.sqrt(inp.D)
    sk = f64(inp.meta["layout_seq_k"][d])
    sv = f64(inp.meta["layout_seq_v"][d])
    P_d = int(inp.prefix_cu[d + 1] - inp.prefix_cu[d])
    b = int(inp.meta["layout_branches"][d])
    out = np.zeros((inp.m, inp.H_q, inp.D))
    lse = np.zeros((inp.m, inp.H_q))
    for i in range(inp.m):
        n = P_d + i + 1
        for h in range(inp.H_q):
            s = scale * (sk[:n, h // G] @ f64(inp.q[b * inp.m + i, h]))
            out[i, h] = softmax(s) @ sv[:n, h // G]
            lse[i, h] = logsumexp(s)
    return out, lse


@pytest.mark.parametrize("case", range(3))
def test_layout_branch_is_a_plain_causal_sequence(case):
    inp = list(small_cases())[case]
    out, lse = oracle.branch_attn(inp)
    for d in range(inp.n_docs):
        b = int(inp.meta["layout_branches"][d])
        ro, rl = causal_sequence_rows(inp, d)
        rows = slice(b * inp.m, (b + 1) * inp.m)
        np.testing.assert_allclose(out[rows], ro, rtol=0, atol=1e-12)
        np.testing.assert_allclose(lse[rows], rl, rtol=0, atol=1e-12)


@pytest.mark.parametrize("case", range(3))
def test_layout_workload_matches_brute_force(case):
    # content branches see the prefix up to their fork (past the vision
    # part) plus their own history; the paged and contiguous prefixes agree
    inp = list(small_cases())[case]
    bo, bl = brute_force(inp)
    out, lse = oracle.branch_attn(inp)
    np.testing.assert_allclose(out, bo, rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse, bl, rtol=0, atol=1e-12)
    inp.prefix_page_table = None
    out2, lse2 = oracle.branch_attn(inp)
    np.testing.assert_array_equal(out, out2)


def test_layout_preset_structure():
    inp = W.make_layout_config()
    V, A = inp.meta["vision_lens"], inp.meta["layout_lens"]
    lay = inp.meta["layout_branches"]
    assert inp.n_docs == 8 and np.all((V >= 1024) & (V <= 3072)) and np.all((A >= 64) & (A <= 512))
    P = np.diff(inp.prefix_cu)
    for d in range(inp.n_docs):
        b = int(lay[d])
        assert inp.branch_prefix_len[b] == V[d] // 16 * 16
        assert inp.branch_len[b] == P[d] + inp.m - V[d] // 16 * 16
        # the layout branch's first private page is a prefix page: shared, not copied
        assert inp.page_table[b, 0] == inp.prefix_page_table[d, V[d] // 16]
        c = np.arange(b + 1, int(inp.branch_cu[d + 1]))
        assert np.all((inp.branch_prefix_len[c] > V[d]) & (inp.branch_prefix_len[c] <= P[d]))


# ------------------------------------------------------------------- GPU --

def _run_gpu(inp):
    import torch
    from paper_2607_18839_gb300 import hpd as H
    d = H.DeviceInputs.from_host(inp)
    op = H.BranchAttn(d)
    out, lse = op()
    torch.cuda.synchronize()
    return out.float().cpu().numpy(), lse.cpu().numpy(), op.errors()


def _compare(out, lse, ro, rl):
    assert np.array_equal(np.isneginf(lse), np.isneginf(rl))
    fin = np.isfinite(rl)
    assert np.max(np.abs(lse[fin] - rl[fin]), initial=0.0) <= LSE_TOL
    assert np.max(np.abs(out - ro)) <= OUT_TOL


@pytest.fixture(scope="module")
def gpu():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_18839_gb300 import build, hpd as H
    build.build()
    H.load()


@pytest.mark.gpu
@pytest.mark.parametrize("case", range(3))
def test_gpu_layout_small_elementwise(gpu, case):
    inp = list(small_cases())[case]
    ro, rl = oracle.branch_attn(inp)
    out, lse, err = _run_gpu(inp)
    assert err == 0
    _compare(out, lse, ro, rl)


@pytest.mark.gpu
def test_gpu_layout_preset_sampled_branches(gpu):
    inp = W.make_layout_config()
    rng = np.random.default_rng(6)
    sel = sorted(set(inp.meta["layout_branches"].tolist()) |
                 set(rng.choice(inp.B, size=12, replace=False).tolist()))
    sel = np.array(sel, np.int32)
    ro, rl = oracle.branch_attn(inp, branch_sel=sel)
    out, lse, err = _run_gpu(inp)
    assert err == 0
    rows = (sel[:, None] * inp.m + np.arange(inp.m)[None, :]).reshape(-1)
    _compare(out[rows], lse[rows], ro[rows], rl[rows])
