"""The seeded input generator: determinism, shapes and structure."""
import numpy as np
import pytest

from paper_2607_18839_gb300 import workloads as W


def test_bf16_rounding_is_nearest_even():
    x = np.array([1.0, 1.0 + 2**-8, 1.0 + 3 * 2**-8, -2.5, 0.0, 3.0e38], dtype=np.float32)
    b = W.f32_to_bf16_bits(x)
    back = W.bf16_bits_to_f32(b)
    # 1 + 2^-8 is a tie between 1 and 1 + 2^-7: even mantissa -> 1.0
    assert back[0] == 1.0 and back[1] == 1.0 and back[2] == 1.0 + 2**-6
    assert back[3] == -2.5 and back[4] == 0.0


@pytest.mark.parametrize("name", ["c1", "c2", "c3"])
def test_configs_are_deterministic_and_well_formed(name):
    a = W.make_config(name)
    b = W.make_config(name)
    assert np.array_equal(a.q, b.q) and np.array_equal(a.page_table, b.page_table)
    assert a.q.shape == (a.B * a.m, a.H_q, a.D)
    assert a.prefix_k.shape == (a.prefix_tokens, a.H_kv, a.D)
    assert a.k_cache.shape == (a.num_pages, W.PAGE, a.H_kv, a.D)
    assert np.all((a.page_table >= 0) & (a.page_table < a.num_pages))
    used = []
    for bb in range(a.B):
        n = (int(a.branch_len[bb]) + W.PAGE - 1) // W.PAGE
        used.extend(a.page_table[bb, :n].tolist())
    assert len(used) == len(set(used))  # no physical page shared between branches


def test_config_shapes_match_the_presets():
    c4 = W.make_config("c4")
    assert c4.n_docs == 32 and c4.B == 32 * 24 and c4.m == 8 and (c4.H_q, c4.H_kv) == (16, 2)
    P = np.diff(c4.prefix_cu)
    assert P.min() >= 1024 and P.max() <= 3072
    c5 = W.make_config("c5")
    s = c5.branch_len - c5.m
    assert s.min() >= 8 and s.max() <= 2048 and c5.B == 256


def test_mix_drafts_rate():
    t = np.arange(40000, dtype=np.int32).reshape(10000, 4) % 32000
    d = W.mix_drafts(t, 32000, 0.7, seed=3)
    rate = np.mean(d == t)
    assert 0.68 < rate < 0.72


def _used_private_pages(inp):
    out = {}
    for b in range(inp.B):
        n = (int(inp.branch_len[b]) + W.PAGE - 1) // W.PAGE
        out[b] = inp.page_table[b, :n].tolist()
    return out


@pytest.mark.parametrize("runs", [False, True])
def test_page_the_prefix_layout(runs):
    base = W.build_inputs([40, 0, 33], [2, 1, 3], [5, 20, 1, 17, 40, 9], 2, 8, 2, 64, seed=3)
    inp = W.page_the_prefix(base, seed=4, extra_pages=3, runs=runs)
    assert inp.num_pages == base.num_pages + 3 + sum((int(p) + 15) // 16 for p in np.diff(base.prefix_cu))
    priv = [pg for pages in _used_private_pages(inp).values() for pg in pages]
    pre = []
    for d in range(inp.n_docs):
        P = int(inp.prefix_cu[d + 1] - inp.prefix_cu[d])
        pages = inp.prefix_page_table[d, :(P + 15) // 16].tolist()
        pre.extend(pages)
        if runs and pages:  # one allocation: consecutive pool pages
            assert pages == list(range(pages[0], pages[0] + len(pages)))
        # the pool pages hold the prefix keys, slot by slot
        for j in range(P):
            assert np.array_equal(inp.k_cache[pages[j // 16], j % 16],
                                  base.prefix_k[int(base.prefix_cu[d]) + j])
    every = priv + pre
    assert len(every) == len(set(every)) and all(0 <= x < inp.num_pages for x in every)
    # the private keys moved with their pages
    for b, pages in _used_private_pages(inp).items():
        old = _used_private_pages(base)[b]
        for a, o in zip(pages, old):
            assert np.array_equal(inp.k_cache[a], base.k_cache[o])


def test_layout_inputs_share_the_prefix_pages_without_copy():
    inp = W.build_layout_inputs([37, 64, 16], [20, 0, 45], [2, 3, 0], [5, 17, 1, 40, 9], 3, 4, 2,
                                64, seed=3)
    V, A = inp.meta["vision_lens"], inp.meta["layout_lens"]
    lay = inp.meta["layout_branches"]
    priv = _used_private_pages(inp)
    content_pages = [pg for b, pages in priv.items() if b not in set(lay.tolist()) for pg in pages]
    assert len(content_pages) == len(set(content_pages))
    for d in range(inp.n_docs):
        P = int(V[d] + A[d])
        b = int(lay[d])
        pre = inp.prefix_page_table[d, :(P + 15) // 16].tolist()
        own = priv[b]
        v16 = int(V[d]) // 16
        # the layout branch's private pages continue the prefix pages from the vision boundary
        assert own[:len(pre) - v16] == pre[v16:]
        assert not set(own) & set(content_pages)
        # its sequence: prefix keys, then the drafts in the slots after P
        seq = inp.meta["layout_seq_k"][d]
        assert seq.shape[0] == P + inp.m
        assert np.array_equal(inp.prefix_k[inp.prefix_cu[d]:inp.prefix_cu[d + 1]], seq[:P])
