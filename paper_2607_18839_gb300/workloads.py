"""Seeded synthetic inputs for one branch-decode step.

This module only draws inputs.  It holds none of the step's arithmetic (no
attention, no softmax, no argmax): it is the single input source shared by
the CUDA path and the oracle.  Everything is numpy; bfloat16 tensors are kept
as their uint16 bit patterns.

Shapes follow the paper's pages (stand-ins for OmniDocBench pages, which are
not available here): a page's shared prefix is its vision tokens plus the
layout branch's tokens (Sec. 3.2 "Visual Encoder", Sec. 3.3), content
branches fork from it, and each branch carries m P-MTP query tokens
(Sec. 3.4).  Paged KV uses 16-token pages in a seeded random physical order.

Presets ``c1`` .. ``c5`` are the five workloads of the branch-decode
benchmark:

c1  one page, prefix 256, 4 branches with suffix 8/16/24/32, m=1, H_q 8 / H_kv 2, D 64
c2  one page, prefix 1,152 (1,024 vision + 128 layout), 16 branches with suffix
    U[16,256], m=4, H_q 16 / H_kv 2, D 128
c3  one page, prefix 4,096, 64 branches with suffix round(lognormal(4.5, 0.8))
    clipped to [1, 1024], m=4, H_q 32 / H_kv 8, D 128
c4  32 pages, prefix U[1024, 3072] each, 24 branches per page with lognormal
    suffixes, m=8, H_q 16 / H_kv 2, D 128, one global page pool
c5  one page, prefix 8,192, 256 branches with suffix
    clip(floor(8 (1 + Pareto(1.5))), 8, 2048), m=4, H_q 32 / H_kv 8, D 128;
    plus acceptance inputs: logits [256, 4, 32000] ~ N(0,1) in bf16

"suffix" s_b is the private history already cached; the branch's private
length is L_b = s_b + m because the step's own m tokens are written to the
cache before attention.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Optional

import numpy as np

PAGE = 16


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bfloat16 (round to nearest, ties to even)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    bias = ((u >> 16) & 1) + 0x7FFF
    return ((u + bias) >> 16).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Widen bfloat16 bit patterns to float32 (exact)."""
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


@dataclass
class BranchDecodeInputs:
    """All inputs of one branch-attention call (host numpy arrays)."""

    n_docs: int
    B: int
    m: int
    H_q: int
    H_kv: int
    D: int
    num_pages: int
    max_pages: int
    q: np.ndarray             # uint16 [B*m, H_q, D]
    prefix_k: np.ndarray      # uint16 [sum P_d, H_kv, D]
    prefix_v: np.ndarray
    prefix_cu: np.ndarray     # int32 [n_docs+1]
    branch_cu: np.ndarray     # int32 [n_docs+1]
    k_cache: np.ndarray       # uint16 [num_pages, 16, H_kv, D]
    v_cache: np.ndarray
    page_table: np.ndarray    # int32 [B, max_pages]
    branch_len: np.ndarray    # int32 [B]
    branch_prefix_len: Optional[np.ndarray] = None  # int32 [B] or None
    # paged prefix: page d's prefix token j is slot j % 16 of pool page
    # prefix_page_table[d, j // 16]; int32 [n_docs, max_prefix_pages] or None
    prefix_page_table: Optional[np.ndarray] = None
    scale: float = 0.0        # 0 -> 1/sqrt(D)
    name: str = "custom"
    meta: dict = field(default_factory=dict)

    @property
    def rows(self) -> int:
        return self.B * self.m

    @property
    def prefix_tokens(self) -> int:
        return int(self.prefix_cu[-1])

    @property
    def max_prefix_len(self) -> int:
        return int(np.max(np.diff(self.prefix_cu))) if self.n_docs else 0

    @property
    def max_prefix_pages(self) -> int:
        return 0 if self.prefix_page_table is None else int(self.prefix_page_table.shape[1])


def _normal_bf16(rng: np.random.Generator, shape, std: float) -> np.ndarray:
    return f32_to_bf16_bits(rng.standard_normal(shape, dtype=np.float32) * np.float32(std))


def build_inputs(
    prefix_lens,
    branches_per_doc,
    suffix_lens,
    m: int,
    H_q: int,
    H_kv: int,
    D: int,
    seed: int,
    *,
    std: float = 0.5,
    branch_prefix_len=None,
    extra_pages: int = 0,
    max_pages: Optional[int] = None,
    scale: float = 0.0,
    name: str = "custom",
) -> BranchDecodeInputs:
    """Draw one workload.

    prefix_lens[d]       shared-prefix length P_d of page d
    branches_per_doc[d]  number of content branches forked from page d
    suffix_lens[b]       cached private history s_b of branch b (L_b = s_b + m)
    branch_prefix_len    optional per-branch fork-position prefix (<= P_d)
    extra_pages          unused pages mixed into the pool
    """
    rng = np.random.default_rng(seed)
    prefix_lens = np.asarray(prefix_lens, dtype=np.int64)
    branches_per_doc = np.asarray(branches_per_doc, dtype=np.int64)
    n_docs = len(prefix_lens)
    assert len(branches_per_doc) == n_docs
    B = int(branches_per_doc.sum())
    suffix_lens = np.asarray(suffix_lens, dtype=np.int64)
    assert len(suffix_lens) == B
    branch_len = (suffix_lens + m).astype(np.int32)
    assert np.all(branch_len >= 0)

    prefix_cu = np.zeros(n_docs + 1, dtype=np.int32)
    prefix_cu[1:] = np.cumsum(prefix_lens)
    branch_cu = np.zeros(n_docs + 1, dtype=np.int32)
    branch_cu[1:] = np.cumsum(branches_per_doc)

    pages_needed = (branch_len.astype(np.int64) + PAGE - 1) // PAGE
    if max_pages is None:
        max_pages = int(max(1, pages_needed.max() if B else 1))
    assert np.all(pages_needed <= max_pages)
    used = int(pages_needed.sum())
    num_pages = max(1, used + extra_pages)
    perm = rng.permutation(num_pages).astype(np.int32)

    page_table = np.zeros((max(B, 0), max_pages), dtype=np.int32)
    cursor = 0
    for b in range(B):
        n = int(pages_needed[b])
        page_table[b, :n] = perm[cursor:cursor + n]
        cursor += n
        # entries past the branch's last page are never read; keep them valid ids
        page_table[b, n:] = rng.integers(0, num_pages, size=max_pages - n)

    T = int(prefix_cu[-1])
    q = _normal_bf16(rng, (B * m, H_q, D), std)
    prefix_k = _normal_bf16(rng, (T, H_kv, D), std)
    prefix_v = _normal_bf16(rng, (T, H_kv, D), std)
    k_cache = _normal_bf16(rng, (num_pages, PAGE, H_kv, D), std)
    v_cache = _normal_bf16(rng, (num_pages, PAGE, H_kv, D), std)

    bpl = None
    if branch_prefix_len is not None:
        bpl = np.asarray(branch_prefix_len, dtype=np.int32)
        assert len(bpl) == B

    return BranchDecodeInputs(
        n_docs=n_docs, B=B, m=m, H_q=H_q, H_kv=H_kv, D=D, num_pages=num_pages,
        max_pages=max_pages, q=q, prefix_k=prefix_k, prefix_v=prefix_v,
        prefix_cu=prefix_cu, branch_cu=branch_cu, k_cache=k_cache, v_cache=v_cache,
        page_table=page_table, branch_len=branch_len, branch_prefix_len=bpl,
        scale=scale, name=name,
        meta=dict(seed=seed, suffix_lens=suffix_lens.astype(np.int32)),
    )


def page_the_prefix(inp: BranchDecodeInputs, seed: int, extra_pages: int = 0,
                    runs: bool = False) -> BranchDecodeInputs:
    """The same workload with every page's prefix moved into the KV pool.

    Page d's prefix occupies ceil(P_d / 16) pool pages.  With ``runs`` they
    are consecutive pool pages (one prefill allocation), the runs and the
    private pages in a seeded random order; otherwise every page, prefix or
    private, lands at a seeded random position.  Slots past P_d in the last
    prefix page hold unrelated finite values.  The contiguous ``prefix_k`` /
    ``prefix_v`` are kept (same keys, for comparisons).
    """
    rng = np.random.default_rng(seed)
    P = np.diff(inp.prefix_cu).astype(np.int64)
    n_pp = (P + PAGE - 1) // PAGE
    max_pp = int(max(1, n_pp.max() if len(n_pp) else 1))
    total = inp.num_pages + int(n_pp.sum()) + extra_pages
    # allocation units: each private page, each extra page, and each page's
    # prefix (one unit of n_pp[d] pages with runs, else n_pp[d] units of one)
    units = [("old", i, 1) for i in range(inp.num_pages)]
    units += [("extra", i, 1) for i in range(extra_pages)]
    for d in range(inp.n_docs):
        if runs:
            units.append(("pre", (d, 0), int(n_pp[d])))
        else:
            units += [("pre", (d, pp), 1) for pp in range(int(n_pp[d]))]
    order = rng.permutation(len(units))
    old_to_new = np.zeros(inp.num_pages, np.int32)
    ppt = rng.integers(0, total, size=(inp.n_docs, max_pp)).astype(np.int32)
    where = 0
    for u in order:
        kind, key, n = units[u]
        if kind == "old":
            old_to_new[key] = where
        elif kind == "pre":
            d, pp0 = key
            ppt[d, pp0:pp0 + n] = np.arange(where, where + n, dtype=np.int32)
        where += n
    assert where == total
    k_cache = _normal_bf16(rng, (total, PAGE, inp.H_kv, inp.D), 0.5)
    v_cache = _normal_bf16(rng, (total, PAGE, inp.H_kv, inp.D), 0.5)
    k_cache[old_to_new] = inp.k_cache
    v_cache[old_to_new] = inp.v_cache
    for d in range(inp.n_docs):
        base = int(inp.prefix_cu[d])
        for pp in range(int(n_pp[d])):
            n = min(PAGE, int(P[d]) - pp * PAGE)
            k_cache[ppt[d, pp], :n] = inp.prefix_k[base + pp * PAGE: base + pp * PAGE + n]
            v_cache[ppt[d, pp], :n] = inp.prefix_v[base + pp * PAGE: base + pp * PAGE + n]
    return BranchDecodeInputs(
        n_docs=inp.n_docs, B=inp.B, m=inp.m, H_q=inp.H_q, H_kv=inp.H_kv, D=inp.D,
        num_pages=total, max_pages=inp.max_pages, q=inp.q, prefix_k=inp.prefix_k,
        prefix_v=inp.prefix_v, prefix_cu=inp.prefix_cu, branch_cu=inp.branch_cu,
        k_cache=k_cache, v_cache=v_cache, page_table=old_to_new[inp.page_table],
        branch_len=inp.branch_len, branch_prefix_len=inp.branch_prefix_len,
        prefix_page_table=ppt, scale=inp.scale,
        name=inp.name + ("-paged-runs" if runs else "-paged"),
        meta=dict(inp.meta, paged_prefix_seed=seed, paged_prefix_runs=runs))


def build_layout_inputs(
    vision_lens,
    layout_lens,
    content_per_doc,
    content_suffix,
    m: int,
    H_q: int,
    H_kv: int,
    D: int,
    seed: int,
    *,
    std: float = 0.5,
    extra_pages: int = 0,
    name: str = "layout",
) -> BranchDecodeInputs:
    """One step in which every page's layout branch decodes beside the
    content branches already forked from it (Sec. 3.3, Algorithm 1).

    Page d's layout sequence is V_d vision tokens, then A_d layout tokens,
    then the layout branch's m drafts of this step; it sits in one run of
    consecutive pool pages (one allocation).  The shared prefix is
    P_d = V_d + A_d (the prefix page table points into that run).  The
    layout branch is branch ``branch_cu[d]``: an ordinary sequence with m
    P-MTP queries whose context is only the page's own tokens, encoded with
    no copy as fork prefix V16_d = 16 floor(V_d / 16) plus private pages =
    the run's pages from V16_d on, L_b = P_d + m - V16_d (its drafts fill the
    slots after P_d of the shared last prefix page, which no content branch
    sees).  Content branch c forks after a layout token: fork prefix f_c
    uniform in [V_d + 1, P_d] (V_d when A_d = 0), private history
    content_suffix[c] + m in scattered pages.  ``meta['layout_seq_k']`` /
    ``['layout_seq_v']`` hold each page's whole sequence (P_d + m tokens).
    """
    rng = np.random.default_rng(seed)
    V = np.asarray(vision_lens, dtype=np.int64)
    A = np.asarray(layout_lens, dtype=np.int64)
    C = np.asarray(content_per_doc, dtype=np.int64)
    n_docs = len(V)
    assert len(A) == n_docs and len(C) == n_docs
    P = V + A
    B = int(n_docs + C.sum())
    content_suffix = np.asarray(content_suffix, dtype=np.int64)
    assert len(content_suffix) == int(C.sum())
    run_pages = (P + m + PAGE - 1) // PAGE
    content_len = (content_suffix + m).astype(np.int64)
    content_pages = (content_len + PAGE - 1) // PAGE
    total = int(run_pages.sum() + content_pages.sum()) + extra_pages
    # allocation units: one run per page's layout sequence, one unit per
    # content page (allocated over time), extra pages; random order
    units = [("run", d, int(run_pages[d])) for d in range(n_docs)]
    units += [("cpage", i, 1) for i in range(int(content_pages.sum()))]
    units += [("extra", i, 1) for i in range(extra_pages)]
    start = {}
    where = 0
    for u in rng.permutation(len(units)):
        kind, key, n = units[u]
        start[(kind, key)] = where
        where += n
    k_cache = _normal_bf16(rng, (total, PAGE, H_kv, D), std)
    v_cache = _normal_bf16(rng, (total, PAGE, H_kv, D), std)

    branch_cu = np.zeros(n_docs + 1, np.int32)
    branch_cu[1:] = np.cumsum(C + 1)
    prefix_cu = np.zeros(n_docs + 1, np.int32)
    prefix_cu[1:] = np.cumsum(P)
    V16 = (V // PAGE) * PAGE
    branch_len = np.zeros(B, np.int32)
    bpl = np.zeros(B, np.int32)
    max_pages = int(max([run_pages[d] - V16[d] // PAGE for d in range(n_docs)] +
                        ([int(content_pages.max())] if len(content_pages) else [1])))
    page_table = rng.integers(0, total, size=(B, max_pages)).astype(np.int32)
    max_pp = int(max(1, ((P + PAGE - 1) // PAGE).max()))
    ppt = rng.integers(0, total, size=(n_docs, max_pp)).astype(np.int32)
    seq_k, seq_v = [], []
    prefix_k = np.zeros((int(P.sum()), H_kv, D), np.uint16)
    prefix_v = np.zeros_like(prefix_k)
    ci = 0
    for d in range(n_docs):
        r0 = start[("run", d)]
        run = np.arange(r0, r0 + run_pages[d], dtype=np.int32)
        n_seq = int(P[d] + m)
        sk = k_cache[run].reshape(-1, H_kv, D)[:n_seq].copy()
        sv = v_cache[run].reshape(-1, H_kv, D)[:n_seq].copy()
        seq_k.append(sk)
        seq_v.append(sv)
        prefix_k[prefix_cu[d]:prefix_cu[d + 1]] = sk[:P[d]]
        prefix_v[prefix_cu[d]:prefix_cu[d + 1]] = sv[:P[d]]
        n_pp = int((P[d] + PAGE - 1) // PAGE)
        ppt[d, :n_pp] = run[:n_pp]
        b = int(branch_cu[d])  # the layout branch
        bpl[b] = V16[d]
        branch_len[b] = n_seq - V16[d]
        own = run[V16[d] // PAGE:]
        page_table[b, :len(own)] = own
        for c in range(int(C[d])):
            b = int(branch_cu[d]) + 1 + c
            bpl[b] = int(rng.integers(V[d] + 1, P[d] + 1)) if A[d] > 0 else int(V[d])
            branch_len[b] = content_len[ci]
            for j in range(int(content_pages[ci])):
                page_table[b, j] = start[("cpage", int(content_pages[:ci].sum()) + j)]
            ci += 1
    q = _normal_bf16(rng, (B * m, H_q, D), std)
    return BranchDecodeInputs(
        n_docs=n_docs, B=B, m=m, H_q=H_q, H_kv=H_kv, D=D, num_pages=total,
        max_pages=max_pages, q=q, prefix_k=prefix_k, prefix_v=prefix_v, prefix_cu=prefix_cu,
        branch_cu=branch_cu, k_cache=k_cache, v_cache=v_cache, page_table=page_table,
        branch_len=branch_len, branch_prefix_len=bpl, prefix_page_table=ppt, name=name,
        meta=dict(seed=seed, layout_branches=branch_cu[:-1].copy(), vision_lens=V.astype(np.int32),
                  layout_lens=A.astype(np.int32), layout_seq_k=seq_k, layout_seq_v=seq_v))


def make_layout_config(seed: int = 1006) -> BranchDecodeInputs:
    """Layout-branch workload: 8 pages, vision U[1024, 3072] tokens, layout
    tokens so far U[64, 512], U[4, 24] content branches per page forked
    after a layout token with lognormal(4.5, 0.8) private histories, m=4,
    H_q 16 / H_kv 2, D 128 (the shapes of the 32-page preset)."""
    rng = np.random.default_rng(seed + 7919)
    V = rng.integers(1024, 3073, size=8)
    A = rng.integers(64, 513, size=8)
    C = rng.integers(4, 25, size=8)
    s = _lognormal_suffix(rng, int(C.sum()))
    return build_layout_inputs(V, A, C, s, 4, 16, 2, 128, seed, name="layout")


def _lognormal_suffix(rng, n):
    return np.clip(np.round(rng.lognormal(4.5, 0.8, size=n)), 1, 1024).astype(np.int64)


def make_config(name: str, seed: Optional[int] = None) -> BranchDecodeInputs:
    """One of the five preset workloads (see module docstring)."""
    cid = int(name.lstrip("c"))
    if seed is None:
        seed = 1000 + cid
    rng = np.random.default_rng(seed + 7919)  # lengths; tensors use ``seed``
    if cid == 1:
        return build_inputs([256], [4], [8, 16, 24, 32], 1, 8, 2, 64, seed, name="c1")
    if cid == 2:
        s = rng.integers(16, 257, size=16)
        return build_inputs([1152], [16], s, 4, 16, 2, 128, seed, name="c2")
    if cid == 3:
        s = _lognormal_suffix(rng, 64)
        return build_inputs([4096], [64], s, 4, 32, 8, 128, seed,
                            max_pages=(1024 + 4 + PAGE - 1) // PAGE, name="c3")
    if cid == 4:
        P = rng.integers(1024, 3073, size=32)
        s = _lognormal_suffix(rng, 32 * 24)
        return build_inputs(P, [24] * 32, s, 8, 16, 2, 128, seed,
                            max_pages=(1024 + 8 + PAGE - 1) // PAGE, name="c4")
    if cid == 5:
        s = np.clip(np.floor(8.0 * (1.0 + rng.pareto(1.5, size=256))), 8, 2048).astype(np.int64)
        return build_inputs([8192], [256], s, 4, 32, 8, 128, seed,
                            max_pages=(2048 + 4 + PAGE - 1) // PAGE, name="c5")
    raise ValueError(f"unknown workload {name!r}")


CONFIG_NAMES = ("c1", "c2", "c3", "c4", "c5")

# Human-readable description of each preset, used in benchmark output.
CONFIG_DESCRIPTIONS = {
    "c1": "1 page, prefix 256, 4 branches (suffix 8/16/24/32), m=1, Hq8/Hkv2, D64",
    "c2": "1 page, prefix 1152, 16 branches (suffix U[16,256]), m=4, Hq16/Hkv2, D128",
    "c3": "1 page, prefix 4096, 64 branches (suffix lognormal(4.5,0.8)), m=4, Hq32/Hkv8, D128",
    "c4": "32 pages, prefix U[1024,3072], 24 branches/page (lognormal), m=8, Hq16/Hkv2, D128",
    "c5": "1 page, prefix 8192, 256 branches (suffix Pareto(1.5,min 8)<=2048), m=4, Hq32/Hkv8, D128",
}


# Branches and P-MTP queries per branch of each preset.
CONFIG_SHAPES = {"c1": (4, 1), "c2": (16, 4), "c3": (64, 4), "c4": (768, 8), "c5": (256, 4)}


def config_shape(name: str) -> dict:
    """{"B": branches, "m": queries per branch} of a preset, without drawing it."""
    B, m = CONFIG_SHAPES[name]
    return {"B": B, "m": m}


def make_logits(B: int, m: int, V: int, seed: int) -> np.ndarray:
    """bf16 logits [B, m, V] drawn N(0, 1)."""
    rng = np.random.default_rng(seed)
    return f32_to_bf16_bits(rng.standard_normal((B, m, V), dtype=np.float32))


def mix_drafts(target_tokens: np.ndarray, V: int, p_match: float, seed: int) -> np.ndarray:
    """Draft tokens: ``target_tokens`` (the caller's row argmax) with
    probability ``p_match`` per position, else a uniform random token."""
    rng = np.random.default_rng(seed)
    target_tokens = np.asarray(target_tokens, dtype=np.int32)
    keep = rng.random(target_tokens.shape) < p_match
    rand = rng.integers(0, V, size=target_tokens.shape, dtype=np.int32)
    return np.where(keep, target_tokens, rand).astype(np.int32)


def accept_inputs(seed: int = 1005, B: int = 256, m: int = 4, V: int = 32000):
    """Logits for the c5 acceptance step (drafts are mixed in by the caller
    from the row argmax it trusts, via :func:`mix_drafts`)."""
    return make_logits(B, m, V, seed)


# ---------------------------------------------------------- paged KV pool --

def make_kv_pool(lengths, m: int, H_kv: int, D: int, num_pages: int, max_pages: int,
                 seed: int):
    """A seeded paged-KV pool: random bf16 caches, each branch's first
    ceil(L_b / 16) logical pages on distinct random physical pages (the rest
    of its table row -1), and the unused page ids, shuffled, on the free
    stack ``free[0:top]``.  Returns a dict of numpy arrays and ``top``."""
    rng = np.random.default_rng(seed)
    lengths = np.asarray(lengths, dtype=np.int32)
    B = lengths.shape[0]
    used = [(int(l) + PAGE - 1) // PAGE for l in lengths]
    if sum(used) > num_pages:
        raise ValueError("pool too small for the lengths")
    perm = rng.permutation(num_pages).astype(np.int32)
    page_table = np.full((B, max_pages), -1, dtype=np.int32)
    at = 0
    for b in range(B):
        page_table[b, :used[b]] = perm[at:at + used[b]]
        at += used[b]
    free = np.zeros(num_pages, dtype=np.int32)
    rest = perm[at:]
    free[:rest.shape[0]] = rest
    shape = (num_pages, PAGE, H_kv, D)
    return dict(
        k_cache=f32_to_bf16_bits(rng.standard_normal(shape, dtype=np.float32) * 0.5),
        v_cache=f32_to_bf16_bits(rng.standard_normal(shape, dtype=np.float32) * 0.5),
        page_table=page_table, branch_len=lengths.copy(), free=free, top=int(rest.shape[0]))


def make_kv_rows(B: int, m: int, H_kv: int, D: int, seed: int):
    """bf16 bits [B, m, H_kv, D] of a step's new keys and values."""
    rng = np.random.default_rng(seed)
    shape = (B, m, H_kv, D)
    return (f32_to_bf16_bits(rng.standard_normal(shape, dtype=np.float32) * 0.5),
            f32_to_bf16_bits(rng.standard_normal(shape, dtype=np.float32) * 0.5))
