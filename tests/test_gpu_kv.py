"""Parity of hpd_kv_append / hpd_kv_rollback with the paged-KV oracle,
bit-exact: caches, page table, lengths, free-page stack and error bits."""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu

from oracle import kv as K
from paper_2607_18839_gb300 import workloads as W


def _dev(st, m):
    import torch
    from paper_2607_18839_gb300 import hpd as H
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    kc = t(st.k_cache.view(np.int16))
    vc = t(st.v_cache.view(np.int16))
    top = torch.tensor([st.top], dtype=torch.int32, device="cuda")
    return H.PagedKV(kc, vc, t(st.page_table), t(st.branch_len), t(st.free), top, m)


def _compare(dv, st, err_expected):
    import torch
    torch.cuda.synchronize()
    assert np.array_equal(dv.branch_len.cpu().numpy(), st.branch_len)
    assert np.array_equal(dv.page_table.cpu().numpy(), st.page_table)
    assert int(dv.free_top.item()) == st.top
    assert np.array_equal(dv.free_pages.cpu().numpy()[:st.top], st.free[:st.top])
    assert np.array_equal(dv.k_cache.cpu().numpy().view(np.uint16), st.k_cache)
    assert np.array_equal(dv.v_cache.cpu().numpy().view(np.uint16), st.v_cache)
    assert dv.errors() == err_expected


def _run(lengths, m, H, D, pages, max_pages, steps, seed, acc_hi=None):
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    p = W.make_kv_pool(lengths, m, H, D, pages, max_pages, seed)
    st = K.KVState(p["k_cache"], p["v_cache"], p["page_table"], p["branch_len"], p["free"], p["top"])
    dv = _dev(st, m)
    B = len(lengths)
    rng = np.random.default_rng(seed + 1)
    err_all = 0
    for s in range(steps):
        kn, vn = W.make_kv_rows(B, m, H, D, seed=seed + 10 + s)
        st, e = K.append(st, kn, vn)
        err_all |= e
        dv.append(torch.from_numpy(kn.view(np.int16)).cuda(), torch.from_numpy(vn.view(np.int16)).cuda())
        _compare(dv, st, err_all)
        acc = rng.integers(-1, (acc_hi or m) + 1, size=B).astype(np.int32)
        st, e = K.rollback(st, acc, m)
        err_all |= e
        dv.rollback(torch.from_numpy(acc).cuda())
        _compare(dv, st, err_all)


def test_c5_like_branches():
    rng = np.random.default_rng(0)
    lengths = np.clip(np.floor(8 * (1 + rng.pareto(1.5, 256))), 8, 600).astype(np.int32)
    _run(lengths, m=4, H=8, D=128, pages=2500, max_pages=48, steps=4, seed=11)


def test_c4_like_branches():
    # 768 branches and 1024 (the largest one-pass scan)
    rng = np.random.default_rng(2)
    lengths = np.clip(np.round(rng.lognormal(4.5, 0.8, 768)), 1, 1024).astype(np.int32)
    _run(lengths, m=8, H=2, D=128, pages=8000, max_pages=70, steps=3, seed=16)
    lengths = rng.integers(0, 40, size=1024).astype(np.int32)
    _run(lengths, m=4, H=2, D=64, pages=5000, max_pages=4, steps=2, seed=17)


def test_many_branches_two_scan_chunks_d64():
    rng = np.random.default_rng(1)
    lengths = rng.integers(2, 70, size=1500).astype(np.int32)
    _run(lengths, m=2, H=2, D=64, pages=9000, max_pages=8, steps=3, seed=12)


def test_m1_all_accepted():
    _run(np.array([0, 15, 16, 17, 31], np.int32), m=1, H=1, D=64, pages=32, max_pages=4,
         steps=3, seed=13, acc_hi=1)


def test_pool_exhausted_and_overlong_branch_change_nothing():
    # 1 free page, 2 needed: the append is refused, then rollback of rows that
    # were never appended is refused as well (branch shorter than m)
    _run(np.array([16, 16, 0], np.int32), m=4, H=1, D=64, pages=3, max_pages=4, steps=1, seed=14)
    _run(np.array([60, 4], np.int32), m=8, H=1, D=64, pages=8, max_pages=4, steps=1, seed=15)
