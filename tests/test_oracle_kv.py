"""Pins of the paged-KV oracle (append before attention, rollback after
acceptance; Algorithm 1).  The oracle is checked against a hand-worked
example, against an independently kept dense copy of every branch's rows,
and against invariants of the page pool."""
import numpy as np
import pytest

from oracle import kv as K
from paper_2607_18839_gb300 import workloads as W


def _state(lengths, m=4, H=2, D=8, pages=64, max_pages=8, seed=0):
    p = W.make_kv_pool(lengths, m, H, D, pages, max_pages, seed)
    return K.KVState(p["k_cache"], p["v_cache"], p["page_table"], p["branch_len"], p["free"],
                     p["top"])


def test_hand_example():
    # branch 0: 14 rows (1 page), branch 1: 16 rows (1 page), branch 2: 0 rows
    st = _state([14, 16, 0], m=4, pages=10, max_pages=4)
    top0, free0 = st.top, st.free.copy()
    assert top0 == 8
    kn, vn = W.make_kv_rows(3, 4, 2, 8, seed=1)
    s1, err = K.append(st, kn, vn)
    assert err == 0
    # new pages: branch 0 needs 1 (rows 14..17), branch 1 needs 1, branch 2 needs 1
    assert s1.top == top0 - 3
    assert list(s1.page_table[:, 1]) == [free0[5], free0[6], -1]
    assert s1.page_table[2, 0] == free0[7]
    assert list(s1.branch_len) == [18, 20, 4]
    # branch 0 row 15 is its new row 1 (page 0 slot 15); row 16 its new row 2
    assert np.array_equal(s1.k_cache[s1.page_table[0, 0], 15], kn[0, 1])
    assert np.array_equal(s1.v_cache[s1.page_table[0, 1], 0], vn[0, 2])
    # accepted: branch 0 one draft (keep 2), branch 1 none (keep 1), branch 2 all (keep 4)
    s2, err = K.rollback(s1, np.array([1, 0, 4], np.int32), 4)
    assert err == 0
    assert list(s2.branch_len) == [16, 17, 4]
    # branch 0 drops its second page (rows 16, 17 rolled back) onto the stack
    assert s2.top == s1.top + 1
    assert s2.free[s1.top] == s1.page_table[0, 1]
    assert s2.page_table[0, 1] == -1 and s2.page_table[1, 1] == s1.page_table[1, 1]


def test_dense_model_and_pool_invariants():
    rng = np.random.default_rng(7)
    B, m, H, D = 9, 3, 2, 8
    lengths = rng.integers(0, 40, size=B)
    st = _state(lengths, m=m, H=H, D=D, pages=96, max_pages=12, seed=3)
    dense = {b: [(st.k_cache[st.page_table[b, p // 16], p % 16].copy(),
                  st.v_cache[st.page_table[b, p // 16], p % 16].copy())
                 for p in range(int(lengths[b]))] for b in range(B)}
    for step in range(6):
        kn, vn = W.make_kv_rows(B, m, H, D, seed=100 + step)
        st, err = K.append(st, kn, vn)
        assert err == 0
        for b in range(B):
            dense[b] += [(kn[b, j], vn[b, j]) for j in range(m)]
        acc = rng.integers(-1, m + 2, size=B).astype(np.int32)
        st, err = K.rollback(st, acc, m)
        assert err == 0
        for b in range(B):
            keep = 0 if acc[b] < 0 else min(int(acc[b]) + 1, m)
            dense[b] = dense[b][:len(dense[b]) - m + keep]
        for b in range(B):
            gk, gv = K.gather(st, b)
            assert len(gk) == len(dense[b]) == st.branch_len[b]
            for (dk, dv), k, v in zip(dense[b], gk, gv):
                assert np.array_equal(dk, k) and np.array_equal(dv, v)
        used = [int(x) for b in range(B) for x in st.page_table[b] if x >= 0]
        assert len(used) == sum(K.pages_of(int(l)) for l in st.branch_len)
        pool = used + [int(x) for x in st.free[:st.top]]
        assert sorted(pool) == list(range(96))


def test_reject_all_restores_state():
    st = _state([5, 31, 32, 0], m=4, pages=40, max_pages=6, seed=5)
    kn, vn = W.make_kv_rows(4, 4, 2, 8, seed=9)
    s1, _ = K.append(st, kn, vn)
    s2, _ = K.rollback(s1, np.full(4, -1, np.int32), 4)
    assert np.array_equal(s2.branch_len, st.branch_len)
    assert np.array_equal(s2.page_table, st.page_table)
    assert s2.top == st.top
    assert sorted(s2.free[:s2.top]) == sorted(st.free[:st.top])


def test_all_or_nothing():
    st = _state([16, 16], m=4, pages=3, max_pages=4, seed=1)  # 1 free page, 2 needed
    kn, vn = W.make_kv_rows(2, 4, 2, 8, seed=2)
    s1, err = K.append(st, kn, vn)
    assert err == K.ERR_POOL
    assert np.array_equal(s1.branch_len, st.branch_len) and s1.top == st.top
    st = _state([62, 0], m=4, pages=8, max_pages=4, seed=1)  # 62 + 4 > 64 rows
    s1, err = K.append(st, kn, vn)
    assert err == K.ERR_BRANCH_LEN and np.array_equal(s1.page_table, st.page_table)
    s1, err = K.rollback(st, np.zeros(2, np.int32), 4)  # branch 1 has fewer than m rows
    assert err == K.ERR_BRANCH_LEN
