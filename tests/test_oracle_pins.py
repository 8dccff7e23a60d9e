"""Pins of the fp64 oracle against facts fixed by the paper and by mathematics.

None of these checks re-uses the oracle's own loops: each one is an
independently written brute force (explicit full mask matrix over all keys of
a page, library softmax), a closed form, an invariant, or a special case that
reduces to textbook attention.  A plausible mistake in the oracle (a dropped
prefix or private term, an off-by-one in the causal rule, a wrong KV-head
grouping, a wrong scale or log base, a transposed page index) fails at least
one of them.

Sec. 3.3 ("Dynamic Branch Forking and Efficient Context Isolation") fixes
which keys a branch sees; Sec. 3.4 and Algorithm 1's verification step fix
the acceptance rule.
"""
import numpy as np
import pytest
from scipy.special import logsumexp, softmax

import oracle
from paper_2607_18839_gb300 import workloads as W

PAGE = W.PAGE


def f64(bits):
    return W.bf16_bits_to_f32(bits).astype(np.float64)


def brute_force(inp):
    """Explicit-mask attention: for every page, one score matrix of all query
    rows against ALL keys stored for that page (its prefix followed by every
    branch's private keys in logical order), masked with -inf where a key is
    not visible to the row, then a library softmax / logsumexp."""
    G = inp.H_q // inp.H_kv
    scale = inp.scale or 1.0 / np.sqrt(inp.D)
    out = np.zeros((inp.rows, inp.H_q, inp.D))
    lse = np.zeros((inp.rows, inp.H_q))
    qf, pk, pv = f64(inp.q), f64(inp.prefix_k), f64(inp.prefix_v)
    kc, vc = f64(inp.k_cache), f64(inp.v_cache)
    for d in range(inp.n_docs):
        p0, p1 = inp.prefix_cu[d], inp.prefix_cu[d + 1]
        b0, b1 = inp.branch_cu[d], inp.branch_cu[d + 1]
        # key table of the page: (owner branch or -1, position, k, v)
        owners, pos, ks, vs = [], [], [], []
        for j in range(p1 - p0):
            owners.append(-1); pos.append(j); ks.append(pk[p0 + j]); vs.append(pv[p0 + j])
        for b in range(b0, b1):
            for j in range(inp.branch_len[b]):
                page = inp.page_table[b, j // PAGE]
                owners.append(b); pos.append(j)
                ks.append(kc[page, j % PAGE]); vs.append(vc[page, j % PAGE])
        owners = np.array(owners, dtype=np.int64)
        pos = np.array(pos, dtype=np.int64)
        if len(ks):
            K = np.stack(ks)  # [n_keys, H_kv, D]
            V = np.stack(vs)
        rows = np.arange(b0 * inp.m, b1 * inp.m)
        if len(rows) == 0:
            continue
        rb = rows // inp.m
        ri = rows % inp.m
        # explicit visibility mask [rows, n_keys]
        pb = (inp.branch_prefix_len[rb] if inp.branch_prefix_len is not None
              else np.full(len(rows), p1 - p0))
        vis = np.zeros((len(rows), len(owners)), dtype=bool)
        if len(owners):
            is_pre = owners[None, :] == -1
            vis |= is_pre & (pos[None, :] < pb[:, None])
            last = inp.branch_len[rb] - inp.m + ri
            vis |= (owners[None, :] == rb[:, None]) & (pos[None, :] <= last[:, None])
        for h in range(inp.H_q):
            g = h // G
            S = np.full((len(rows), len(owners)), -np.inf)
            if len(owners):
                S_full = scale * (qf[rows, h, :] @ K[:, g, :].T)
                S = np.where(vis, S_full, -np.inf)
            for r in range(len(rows)):
                if not vis[r].any():
                    out[rows[r], h] = 0.0
                    lse[rows[r], h] = -np.inf
                    continue
                w = softmax(S[r])
                out[rows[r], h] = w @ V[:, g, :]
                lse[rows[r], h] = logsumexp(S[r])
    return out, lse


def tiny_cases():
    """Small workloads spanning the structure: several pages, uneven branch
    counts, private lengths below m, zero, and exactly on page boundaries,
    per-branch fork prefixes, an empty prefix, a page with no branches."""
    yield W.build_inputs([7], [3], [0, 5, 16], 2, 4, 2, 8, seed=1)
    yield W.build_inputs([20, 3], [2, 2], [1, 30, 15, 0], 3, 6, 3, 16, seed=2, extra_pages=3)
    yield W.build_inputs([0, 9, 33], [1, 2, 2], [4, 0, 17, 31, 2], 4, 4, 1, 8, seed=3,
                         branch_prefix_len=[0, 9, 4, 33, 0])
    yield W.build_inputs([12, 5], [0, 3], [3, 9, 40], 1, 8, 2, 4, seed=4)
    yield W.build_inputs([16], [2], [0, 0], 1, 2, 2, 8, seed=5)  # m=1, empty suffix
    yield W.make_config("c1")


@pytest.mark.parametrize("case", list(range(6)))
def test_oracle_matches_explicit_mask_brute_force(case):
    inp = list(tiny_cases())[case]
    out, lse = oracle.branch_attn(inp)
    bo, bl = brute_force(inp)
    assert np.array_equal(np.isinf(lse), np.isinf(bl))
    fin = np.isfinite(bl)
    np.testing.assert_allclose(lse[fin], bl[fin], rtol=0, atol=1e-12)
    np.testing.assert_allclose(out, bo, rtol=0, atol=1e-12)


def _visible_count(inp, b, i):
    d = int(np.searchsorted(inp.branch_cu, b, side="right") - 1)
    pb = (inp.branch_prefix_len[b] if inp.branch_prefix_len is not None
          else inp.prefix_cu[d + 1] - inp.prefix_cu[d])
    return int(pb) + max(0, int(inp.branch_len[b]) - inp.m + i + 1), d, int(pb)


def test_zero_query_gives_mean_of_visible_values_and_log_count():
    # Q = 0 makes every visible score 0: weights are uniform, so out is the
    # plain mean of the visible V rows and lse = ln(#visible) exactly.
    inp = W.build_inputs([10, 21], [2, 3], [0, 3, 17, 33, 1], 3, 4, 2, 8, seed=11,
                         branch_prefix_len=[10, 6, 0, 21, 13])
    inp.q[:] = 0
    out, lse = oracle.branch_attn(inp)
    vc, pv = f64(inp.v_cache), f64(inp.prefix_v)
    G = inp.H_q // inp.H_kv
    for b in range(inp.B):
        for i in range(inp.m):
            n, d, pb = _visible_count(inp, b, i)
            row = b * inp.m + i
            for h in range(inp.H_q):
                g = h // G
                if n == 0:
                    assert lse[row, h] == -np.inf and np.all(out[row, h] == 0)
                    continue
                vals = [pv[inp.prefix_cu[d] + j, g] for j in range(pb)]
                for j in range(inp.branch_len[b] - inp.m + i + 1):
                    vals.append(vc[inp.page_table[b, j // PAGE], j % PAGE, g])
                assert abs(lse[row, h] - np.log(n)) < 1e-13
                np.testing.assert_allclose(out[row, h], np.mean(vals, axis=0), atol=1e-13)


def test_constant_values_give_that_value():
    inp = W.build_inputs([13], [3], [2, 9, 40], 2, 4, 2, 8, seed=12)
    c = W.f32_to_bf16_bits(np.linspace(-1, 1, inp.D, dtype=np.float32))
    inp.prefix_v[:] = c
    inp.v_cache[:] = c
    out, _ = oracle.branch_attn(inp)
    np.testing.assert_allclose(out, np.broadcast_to(f64(c), out.shape), atol=1e-13)


def test_empty_suffix_single_query_is_plain_prefix_attention():
    # L_b = 0 with m = 1: the step sees no private key, so each branch reduces
    # to textbook single-query attention over its page's prefix.
    inp = W.build_inputs([37, 5], [2, 1], [0, 0, 0], 1, 6, 3, 16, seed=13)
    inp.branch_len[:] = 0
    out, lse = oracle.branch_attn(inp)
    scale = 1.0 / np.sqrt(inp.D)
    q, pk, pv = f64(inp.q), f64(inp.prefix_k), f64(inp.prefix_v)
    for b in range(inp.B):
        d = int(np.searchsorted(inp.branch_cu, b, side="right") - 1)
        K = pk[inp.prefix_cu[d]:inp.prefix_cu[d + 1]]
        V = pv[inp.prefix_cu[d]:inp.prefix_cu[d + 1]]
        for h in range(inp.H_q):
            g = h // (inp.H_q // inp.H_kv)
            s = scale * K[:, g, :] @ q[b, h]
            np.testing.assert_allclose(out[b, h], softmax(s) @ V[:, g, :], atol=1e-13)
            assert abs(lse[b, h] - logsumexp(s)) < 1e-12


def test_two_keys_closed_form_scale_and_natural_log():
    # One prefix key and one private key, D = 4, values exact in bf16.
    # s1 = <q,k1>/sqrt(4), s2 = <q,k2>/2; out = sigmoid(s1-s2) v1 + sigmoid(s2-s1) v2,
    # lse = ln(e^s1 + e^s2).
    inp = W.build_inputs([1], [1], [0], 1, 1, 1, 4, seed=14)
    bf = W.f32_to_bf16_bits
    inp.q[0, 0] = bf(np.array([1.0, 2.0, 0.0, -1.0], dtype=np.float32))
    inp.prefix_k[0, 0] = bf(np.array([0.5, 0.5, 0.0, 0.0], dtype=np.float32))  # <q,k1> = 1.5
    inp.prefix_v[0, 0] = bf(np.array([1.0, 0.0, 0.0, 0.0], dtype=np.float32))
    page = inp.page_table[0, 0]
    inp.k_cache[page, 0, 0] = bf(np.array([0.0, 0.0, 4.0, -2.0], dtype=np.float32))  # <q,k2> = 2
    inp.v_cache[page, 0, 0] = bf(np.array([0.0, 3.0, 0.0, 0.0], dtype=np.float32))
    out, lse = oracle.branch_attn(inp)
    s1, s2 = 1.5 / 2.0, 2.0 / 2.0
    w1 = 1.0 / (1.0 + np.exp(s2 - s1))
    np.testing.assert_allclose(out[0, 0], [w1, 3.0 * (1 - w1), 0.0, 0.0], atol=1e-15)
    assert abs(lse[0, 0] - np.log(np.exp(s1) + np.exp(s2))) < 1e-15


def test_gqa_groups_contiguous_query_heads():
    # Q = 0 and V constant per KV head: query head h must return KV head h // G.
    inp = W.build_inputs([8], [2], [3, 5], 2, 8, 2, 8, seed=15)
    inp.q[:] = 0
    for g in range(inp.H_kv):
        val = W.f32_to_bf16_bits(np.full(inp.D, float(g + 1), dtype=np.float32))
        inp.prefix_v[:, g] = val
        inp.v_cache[:, :, g] = val
    out, _ = oracle.branch_attn(inp)
    for h in range(inp.H_q):
        np.testing.assert_allclose(out[:, h], float(h // 4 + 1), rtol=0, atol=1e-14)


def test_no_visible_key_gives_zero_and_minus_inf():
    inp = W.build_inputs([4], [1], [0], 3, 2, 1, 8, seed=16, branch_prefix_len=[0])
    inp.branch_len[:] = 1  # only the last query sees one private key
    out, lse = oracle.branch_attn(inp)
    assert np.all(lse[0:2] == -np.inf) and np.all(out[0:2] == 0)
    assert np.all(np.isfinite(lse[2]))
    v0 = f64(inp.v_cache[inp.page_table[0, 0], 0, 0])
    np.testing.assert_allclose(out[2], np.broadcast_to(v0, out[2].shape), atol=1e-13)


def test_permuting_branches_permutes_outputs():
    inp = W.build_inputs([30], [5], [3, 18, 0, 33, 9], 3, 4, 2, 8, seed=17)
    out, lse = oracle.branch_attn(inp)
    perm = np.array([3, 0, 4, 1, 2])
    rows = (perm[:, None] * inp.m + np.arange(inp.m)[None, :]).reshape(-1)
    p = W.BranchDecodeInputs(**{**inp.__dict__})
    p.q = inp.q[rows].copy()
    p.page_table = inp.page_table[perm].copy()
    p.branch_len = inp.branch_len[perm].copy()
    out2, lse2 = oracle.branch_attn(p)
    np.testing.assert_array_equal(out2, out[rows])
    np.testing.assert_array_equal(lse2, lse[rows])


def test_permuting_physical_pages_leaves_outputs_unchanged():
    inp = W.build_inputs([19, 7], [2, 2], [40, 2, 17, 30], 2, 4, 2, 8, seed=18, extra_pages=5)
    out, lse = oracle.branch_attn(inp)
    rng = np.random.default_rng(0)
    perm = rng.permutation(inp.num_pages)  # new id of old page p is perm[p]
    p = W.BranchDecodeInputs(**{**inp.__dict__})
    p.k_cache = np.empty_like(inp.k_cache); p.k_cache[perm] = inp.k_cache
    p.v_cache = np.empty_like(inp.v_cache); p.v_cache[perm] = inp.v_cache
    p.page_table = perm[inp.page_table].astype(np.int32)
    out2, lse2 = oracle.branch_attn(p)
    np.testing.assert_array_equal(out2, out)
    np.testing.assert_array_equal(lse2, lse)


def test_causality_among_the_m_queries():
    # Perturbing private key j changes exactly the queries i with j <= L - m + i.
    inp = W.build_inputs([6], [1], [5], 4, 2, 1, 8, seed=19)
    L, m = int(inp.branch_len[0]), inp.m
    out0, _ = oracle.branch_attn(inp)
    for j in range(L):
        p = W.BranchDecodeInputs(**{**inp.__dict__})
        p.k_cache = inp.k_cache.copy(); p.v_cache = inp.v_cache.copy()
        page = inp.page_table[0, j // PAGE]
        p.k_cache[page, j % PAGE] = W.f32_to_bf16_bits(np.full((1, inp.D), 1.5, np.float32))
        p.v_cache[page, j % PAGE] = W.f32_to_bf16_bits(np.full((1, inp.D), -2.0, np.float32))
        out1, _ = oracle.branch_attn(p)
        for i in range(m):
            changed = not np.array_equal(out1[i], out0[i])
            assert changed == (j <= L - m + i), (j, i)


def test_branch_subset_matches_full_run():
    inp = W.build_inputs([25, 9], [3, 2], [3, 18, 0, 33, 9], 2, 4, 2, 8, seed=20)
    out, lse = oracle.branch_attn(inp)
    sel = np.array([4, 1])
    o2, l2 = oracle.branch_attn(inp, branch_sel=sel)
    rows = (sel[:, None] * inp.m + np.arange(inp.m)).reshape(-1)
    np.testing.assert_array_equal(o2[rows], out[rows])
    np.testing.assert_array_equal(l2[rows], lse[rows])
    assert np.all(np.isnan(np.delete(o2, rows, axis=0)))


# ---------------------------------------------------------------- acceptance


def _logits(rows):
    return W.f32_to_bf16_bits(np.asarray(rows, dtype=np.float32))


def test_accept_closed_forms():
    # B=3 branches, m=3, V=5.  Row argmaxes are chosen by construction.
    lg = _logits([
        [[0, 9, 1, 2, 3], [5, 0, 0, 0, 0], [0, 0, 0, 0, 7]],   # argmax 1, 0, 4
        [[0, 0, 3, 0, 0], [1, 1, 1, 8, 1], [2, 0, 0, 0, 0]],   # argmax 2, 3, 0
        [[4, 4, 1, 4, 0], [0, -1, -1, 0, -2], [-3, -3, -3, -3, -3]],  # ties -> 0, 0, 0
    ])
    drafts = np.array([[1, 0, 4],     # all right -> 3
                       [1, 3, 0],     # first wrong -> 0
                       [0, 1, 0]])    # second wrong -> 1
    tok, acc = oracle.pmtp_accept(lg, drafts)
    np.testing.assert_array_equal(tok, [[1, 0, 4], [2, 3, 0], [0, 0, 0]])
    np.testing.assert_array_equal(acc, [3, 0, 1])


def test_accept_ties_lowest_index_and_nan_ignored():
    nan = np.float32(np.nan)
    lg = _logits([[[1, 2, 2, 2], [nan, 1, 3, 3], [nan, nan, nan, nan], [-np.inf, -np.inf, 0, 0]]])
    tok, acc = oracle.pmtp_accept(lg, np.array([[1, 2, 0, 2]]))
    np.testing.assert_array_equal(tok, [[1, 2, 0, 2]])
    assert acc[0] == 4


def test_accept_matches_numpy_argmax_brute_force():
    rng = np.random.default_rng(21)
    B, m, V = 7, 5, 97
    # coarse values force many ties; np.argmax returns the first maximum
    vals = rng.integers(-4, 5, size=(B, m, V)).astype(np.float32) * 0.25
    lg = _logits(vals)
    ref_tok = np.argmax(W.bf16_bits_to_f32(lg).reshape(B, m, V), axis=-1)
    drafts = np.where(rng.random((B, m)) < 0.6, ref_tok, rng.integers(0, V, (B, m)))
    tok, acc = oracle.pmtp_accept(lg, drafts)
    np.testing.assert_array_equal(tok, ref_tok)
    for b in range(B):
        k = 0
        while k < m and drafts[b, k] == ref_tok[b, k]:
            k += 1
        assert acc[b] == k


@pytest.mark.parametrize("case", list(range(6)))
def test_paged_prefix_matches_brute_force_on_the_same_keys(case):
    # The prefix moved into the pool (own pages, random physical order, the
    # contiguous buffers kept) must give the brute-force result over the
    # contiguous keys; with the contiguous buffers wiped it must not change,
    # so the paged mode reads the pool through the prefix page table.
    inp = W.page_the_prefix(list(tiny_cases())[case], seed=70 + case, extra_pages=2)
    bo, bl = brute_force(inp)
    inp.prefix_k = np.full_like(inp.prefix_k, 0x7FC0)  # NaN bits: must never be read
    inp.prefix_v = np.full_like(inp.prefix_v, 0x7FC0)
    out, lse = oracle.branch_attn(inp)
    assert np.array_equal(np.isinf(lse), np.isinf(bl))
    fin = np.isfinite(bl)
    np.testing.assert_allclose(lse[fin], bl[fin], rtol=0, atol=1e-12)
    np.testing.assert_allclose(out, bo, rtol=0, atol=1e-12)


def test_paged_prefix_follows_the_table():
    # Swapping the first two prefix pages in the table moves keys across the
    # fork limits (16 and 8: only page 0 visible), which changes what the
    # branches see; swapping the pool pages back restores it exactly.
    inp = W.page_the_prefix(W.build_inputs([40], [3], [4, 9, 20], 2, 4, 2, 8, seed=8,
                                           branch_prefix_len=[16, 16, 8]), seed=9)
    o0, _ = oracle.branch_attn(inp)
    a, b = inp.prefix_page_table[0, 0], inp.prefix_page_table[0, 1]
    inp.prefix_page_table[0, [0, 1]] = [b, a]
    o1, _ = oracle.branch_attn(inp)
    assert not np.allclose(o0, o1)
    for cache in (inp.k_cache, inp.v_cache):
        cache[[a, b]] = cache[[b, a]]
    o2, _ = oracle.branch_attn(inp)
    np.testing.assert_array_equal(o0, o2)
