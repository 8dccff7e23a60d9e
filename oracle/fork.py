"""Oracle of fork detection and child branches after verification (test
infrastructure; Algorithm 1, Sec. 3.3).

Plain Python, written from the method: a layout branch emits its accepted
drafts and the correction token, t*_{b,0..e_b-1} with e_b = min(n_acc + 1, m)
(none when n_acc < 0); each emitted fork token at index i (prefix position
layout_pos[b] + i) spawns a child of the same page that sees the page prefix
up to and including the fork token and has no private keys yet.  The new
branch set lists every page's old branches, then its children by parent and
index.

Only tests, ``__graft_entry__.smoke()`` and bench.py's baseline legs use this
module.  Nothing here shares code with the CUDA library.
"""
import numpy as np

ERR_BRANCH_CU = 0x2
ERR_FORK_CAP = 0x100


def fork_children(out_tokens, accepted_len, is_layout, layout_pos, fork_token, branch_cu,
                  branch_prefix_len, branch_len, page_table, cap):
    """Returns (dict of new arrays, error bits); the arrays are None on error."""
    B, m = out_tokens.shape
    n_docs = len(branch_cu) - 1
    if branch_cu[0] != 0 or branch_cu[-1] != B or any(
            branch_cu[d] > branch_cu[d + 1] for d in range(n_docs)):
        return None, ERR_BRANCH_CU
    rows = []  # (parent or -1 - parent, branch_len, prefix_len, page row)
    new_cu = [0]
    for d in range(n_docs):
        olds = list(range(branch_cu[d], branch_cu[d + 1]))
        for b in olds:
            pl = -1 if branch_prefix_len is None else int(branch_prefix_len[b])
            rows.append((b, int(branch_len[b]), pl, page_table[b].copy()))
        for b in olds:
            if is_layout is not None and not is_layout[b]:
                continue
            n = int(accepted_len[b])
            emitted = 0 if n < 0 else min(n + 1, m)
            for i in range(emitted):
                if out_tokens[b, i] == fork_token:
                    rows.append((-1 - b, 0, int(layout_pos[b]) + i + 1,
                                 np.full(page_table.shape[1], -1, np.int32)))
        new_cu.append(len(rows))
    if len(rows) > cap:
        return None, ERR_FORK_CAP
    return dict(
        new_B=len(rows),
        branch_cu=np.array(new_cu, np.int32),
        parent=np.array([r[0] for r in rows], np.int32),
        branch_len=np.array([r[1] for r in rows], np.int32),
        branch_prefix_len=np.array([r[2] for r in rows], np.int32),
        page_table=np.stack([r[3] for r in rows]).astype(np.int32) if rows else
        np.zeros((0, page_table.shape[1]), np.int32)), 0
