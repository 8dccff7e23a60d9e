"""Oracle of the paged private KV around a decode step (test infrastructure).

Plain Python over numpy arrays, written from Algorithm 1: the step's tokens
are written to the branch's paged cache before attention (WriteKV), and after
the verification the branch keeps what was accepted.  The printed length
update of Algorithm 1 is garbled; the reading taken: of the step's m rows,
keep the first n_acc + 1 (at most m; none when n_acc < 0) and roll back the
others.  Free pages form a stack ``free[0:top]``; page ids are handed out and
returned in branch order, all or nothing.

Only tests, ``__graft_entry__.smoke()`` and bench.py's baseline legs use
this module.  Nothing here shares code with the CUDA library.
"""
from dataclasses import dataclass, replace

import numpy as np

PAGE = 16
ERR_BRANCH_LEN = 0x4
ERR_POOL = 0x80


@dataclass
class KVState:
    k_cache: np.ndarray     # uint16 (bf16 bits) [num_pages][16][H_kv][D]
    v_cache: np.ndarray
    page_table: np.ndarray  # int32 [B][max_pages]
    branch_len: np.ndarray  # int32 [B]
    free: np.ndarray        # int32 [num_pages], entries [0, top) are free ids
    top: int

    def copy(self):
        return replace(self, k_cache=self.k_cache.copy(), v_cache=self.v_cache.copy(),
                       page_table=self.page_table.copy(), branch_len=self.branch_len.copy(),
                       free=self.free.copy())


def pages_of(n: int) -> int:
    return (n + PAGE - 1) // PAGE


def append(st: KVState, k_new: np.ndarray, v_new: np.ndarray):
    """Append branch b's m rows (k_new / v_new [B][m][H_kv][D]) at positions
    [L_b, L_b + m).  Returns (new state, error bits)."""
    s = st.copy()
    B, m = k_new.shape[0], k_new.shape[1]
    cap = s.page_table.shape[1] * PAGE
    L = [int(x) for x in s.branch_len]
    if any(l < 0 or l + m > cap for l in L):
        return s, ERR_BRANCH_LEN
    need = [pages_of(L[b] + m) - pages_of(L[b]) for b in range(B)]
    total = sum(need)
    if total > s.top or s.top > s.free.shape[0]:
        return s, ERR_POOL
    nxt = s.top - total  # branch 0 takes the deepest of the popped entries
    for b in range(B):
        for i in range(need[b]):
            s.page_table[b, pages_of(L[b]) + i] = s.free[nxt]
            nxt += 1
    s.top -= total
    for b in range(B):
        for j in range(m):
            pos = L[b] + j
            page = s.page_table[b, pos // PAGE]
            s.k_cache[page, pos % PAGE] = k_new[b, j]
            s.v_cache[page, pos % PAGE] = v_new[b, j]
        s.branch_len[b] = L[b] + m
    return s, 0


def rollback(st: KVState, accepted_len: np.ndarray, m: int):
    """Keep min(n_acc + 1, m) of each branch's last m rows (none when
    n_acc < 0); push the pages past the new length in branch order."""
    s = st.copy()
    B = s.branch_len.shape[0]
    cap = s.page_table.shape[1] * PAGE
    L = [int(x) for x in s.branch_len]
    if any(l < m or l > cap for l in L):
        return s, ERR_BRANCH_LEN
    new = []
    for b in range(B):
        n = int(accepted_len[b])
        keep = 0 if n < 0 else min(n + 1, m)
        new.append(L[b] - m + keep)
    total = sum(pages_of(L[b]) - pages_of(new[b]) for b in range(B))
    if s.top < 0 or s.top + total > s.free.shape[0]:
        return s, ERR_POOL
    for b in range(B):
        for i in range(pages_of(new[b]), pages_of(L[b])):
            s.free[s.top] = s.page_table[b, i]
            s.page_table[b, i] = -1
            s.top += 1
        s.branch_len[b] = new[b]
    return s, 0


def gather(st: KVState, b: int):
    """Branch b's private rows in order, read through its page table."""
    rows_k, rows_v = [], []
    for pos in range(int(st.branch_len[b])):
        page = st.page_table[b, pos // PAGE]
        rows_k.append(st.k_cache[page, pos % PAGE])
        rows_v.append(st.v_cache[page, pos % PAGE])
    return rows_k, rows_v
