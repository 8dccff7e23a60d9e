"""Fork detection and child branches (Algorithm 1, Sec. 3.3): pins of the
oracle (hand-worked example, invariants) and bit-exact parity of
hpd_fork_children with it."""
import numpy as np
import pytest

from oracle import fork as F

FORK = 151666  # any token id serves as the fork token


def _case(rng, n_docs, per_doc, m, max_pages, p_fork):
    counts = rng.integers(0, per_doc + 1, size=n_docs)
    branch_cu = np.concatenate([[0], np.cumsum(counts)]).astype(np.int32)
    B = int(branch_cu[-1])
    tok = rng.integers(0, 1000, size=(B, m)).astype(np.int32)
    tok[rng.random((B, m)) < p_fork] = FORK
    acc = rng.integers(-1, m + 1, size=B).astype(np.int32)
    is_layout = np.zeros(B, np.int32)
    for d in range(n_docs):  # first branch of a page is its layout branch
        if counts[d]:
            is_layout[branch_cu[d]] = 1
    layout_pos = rng.integers(0, 3000, size=B).astype(np.int32)
    bpl = rng.integers(0, 3000, size=B).astype(np.int32)
    blen = rng.integers(0, 200, size=B).astype(np.int32)
    pt = rng.integers(0, 5000, size=(B, max_pages)).astype(np.int32)
    return tok, acc, is_layout, layout_pos, branch_cu, bpl, blen, pt


def test_hand_example():
    # page 0: branches 0 (layout), 1; page 1: branch 2 (layout)
    tok = np.array([[5, FORK, 7, FORK], [FORK, 1, 2, 3], [FORK, 9, 9, 9]], np.int32)
    acc = np.array([2, 4, 0], np.int32)  # branch 0 emits 3 tokens, branch 2 emits 1
    is_layout = np.array([1, 0, 1], np.int32)
    layout_pos = np.array([100, 0, 40], np.int32)
    cu = np.array([0, 2, 3], np.int32)
    pt = np.arange(6, dtype=np.int32).reshape(3, 2)
    new, err = F.fork_children(tok, acc, is_layout, layout_pos, FORK, cu, None,
                               np.array([10, 11, 12], np.int32), pt, cap=8)
    assert err == 0 and new["new_B"] == 5
    # page 0: old 0, old 1, child of 0 at index 1 (prefix 100 + 1 + 1); the
    # fork token at index 3 was not emitted; page 1: old 2, child of 2 (40 + 1)
    assert list(new["branch_cu"]) == [0, 3, 5]
    assert list(new["parent"]) == [0, 1, -1, 2, -3]
    assert list(new["branch_prefix_len"]) == [-1, -1, 102, -1, 41]
    assert list(new["branch_len"]) == [10, 11, 0, 12, 0]
    assert (new["page_table"][2] == -1).all() and (new["page_table"][3] == pt[2]).all()


def test_invariants_and_capacity():
    rng = np.random.default_rng(3)
    tok, acc, lay, pos, cu, bpl, blen, pt = _case(rng, 7, 9, 4, 3, 0.3)
    new, err = F.fork_children(tok, acc, lay, pos, FORK, cu, bpl, blen, pt, cap=10_000)
    assert err == 0
    B = len(blen)
    olds = new["parent"][new["parent"] >= 0]
    assert sorted(olds) == list(range(B))
    n_child = int((new["parent"] < 0).sum())
    expect = sum(int(np.sum(tok[b, :min(acc[b] + 1, 4)] == FORK)) for b in range(B)
                 if lay[b] and acc[b] >= 0)
    assert n_child == expect and new["new_B"] == B + n_child
    for d in range(len(cu) - 1):  # every child lands in its parent's page
        for i in range(new["branch_cu"][d], new["branch_cu"][d + 1]):
            par = new["parent"][i]
            b = par if par >= 0 else -1 - par
            assert cu[d] <= b < cu[d + 1]
    _, err = F.fork_children(tok, acc, lay, pos, FORK, cu, bpl, blen, pt, cap=B + n_child - 1)
    assert err == F.ERR_FORK_CAP
    _, err = F.fork_children(tok, acc, lay, pos, FORK, np.array([0, 5, 3, B], np.int32)
                             if B > 5 else np.array([0, 1, 0, B], np.int32), bpl, blen, pt, cap=10_000)
    assert err == F.ERR_BRANCH_CU


def _gpu(args, cap):
    import torch
    from paper_2607_18839_gb300 import hpd as H
    tok, acc, lay, pos, cu, bpl, blen, pt = args
    t = lambda a: None if a is None else torch.from_numpy(np.ascontiguousarray(a)).cuda()
    new = H.fork_children(t(tok), t(acc), t(lay), t(pos), FORK, t(cu), t(bpl), t(blen), t(pt), cap)
    torch.cuda.synchronize()
    err = int(new["workspace"][:4].view(torch.int32).item())
    return {k: v.cpu().numpy() for k, v in new.items() if k != "workspace"}, err


@pytest.mark.gpu
@pytest.mark.parametrize("n_docs,per_doc,m,p_fork,layout", [
    (1, 16, 4, 0.2, True), (32, 24, 8, 0.05, True), (700, 3, 2, 0.5, False), (3, 0, 4, 0.3, True)])
def test_gpu_parity(n_docs, per_doc, m, p_fork, layout):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    rng = np.random.default_rng(n_docs * 10 + m)
    case = list(_case(rng, n_docs, per_doc, m, 5, p_fork))
    if not layout:
        case[2] = None
    cap = int(case[4][-1]) * (m + 1) + 1
    ref, err = F.fork_children(*case[:4], FORK, *case[4:], cap=cap)
    got, gerr = _gpu(case, cap)
    assert gerr == err == 0
    nb = ref["new_B"]
    assert int(got["new_B"][0]) == nb
    assert np.array_equal(got["branch_cu"], ref["branch_cu"])
    for k in ("parent", "branch_len", "branch_prefix_len", "page_table"):
        assert np.array_equal(got[k][:nb], ref[k]), k


@pytest.mark.gpu
def test_gpu_capacity_and_bad_offsets():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    rng = np.random.default_rng(5)
    case = list(_case(rng, 4, 6, 4, 2, 0.5))
    ref, _ = F.fork_children(*case[:4], FORK, *case[4:], cap=10_000)
    B = int(case[4][-1])
    got, err = _gpu(case, max(B, ref["new_B"] - 1))
    assert err == F.ERR_FORK_CAP and int(got["new_B"][0]) == -1
    bad = list(case)
    bad[4] = np.array([0, 3, 1, 4, B], np.int32)
    got, err = _gpu(bad, 10_000)
    assert err == F.ERR_BRANCH_CU and int(got["new_B"][0]) == -1
