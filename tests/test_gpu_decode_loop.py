"""Several decode iterations of Algorithm 1 on the GPU against the oracle.

Each iteration writes the step's K/V rows into the paged private cache
(hpd_kv_append), runs the step in one call (hpd_decode_step: the attention
over the shared prefix and the grown private histories, and the greedy
acceptance), keeps the accepted rows (hpd_kv_rollback), and at the end the
layout branches' emitted tokens are scanned for the fork token
(hpd_fork_children).  The device state is carried from call to call exactly
as a decoder would carry it; the oracle replays the same iterations on the
host.  Attention within the parity tolerances, everything else bit-exact.
"""
import dataclasses

import numpy as np
import pytest

import oracle
from oracle import fork as F
from oracle import kv as K
from paper_2607_18839_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

V = 4096
FORK = V - 1


@pytest.fixture(scope="module")
def hpd():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_18839_gb300 import build, hpd as H
    build.build()
    H.load()
    return H


def bits(x):
    return torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).cuda()


def i32(x):
    return torch.from_numpy(np.ascontiguousarray(x, dtype=np.int32)).cuda()


@pytest.mark.parametrize("iters,seed", [(4, 700), (3, 701)])
def test_decode_loop_matches_the_oracle(hpd, iters, seed):
    m, H_q, H_kv, D = 4, 16, 2, 128
    # two pages (prefixes 512 and 300 tokens) with 3 and 2 content branches;
    # the first branch of each page plays its layout branch for the fork scan
    base = W.build_inputs([512, 300], [3, 2], [40, 0, 17, 100, 63], m, H_q, H_kv, D, seed=seed)
    B = base.B
    hist = base.meta["suffix_lens"]
    pool = W.make_kv_pool(hist, m, H_kv, D, num_pages=64, max_pages=16, seed=seed + 1)
    st = K.KVState(pool["k_cache"], pool["v_cache"], pool["page_table"], pool["branch_len"],
                   pool["free"], pool["top"])
    kv = hpd.PagedKV(bits(st.k_cache), bits(st.v_cache), i32(st.page_table), i32(st.branch_len),
                     i32(st.free), i32([st.top]), m)
    rng = np.random.default_rng(seed + 2)
    prefix_k, prefix_v = bits(base.prefix_k).view(torch.bfloat16), bits(base.prefix_v).view(torch.bfloat16)
    tok = torch.empty((B, m), dtype=torch.int32, device="cuda")
    acc = torch.empty((B,), dtype=torch.int32, device="cuda")
    for it in range(iters):
        # WriteKV: the step's rows go to the cache before the attention
        kn, vn = W.make_kv_rows(B, m, H_kv, D, seed=seed + 10 + it)
        st, e = K.append(st, kn, vn)
        assert e == 0
        kv.append(bits(kn), bits(vn))
        # the step: queries of the m P-MTP tokens, logits and drafts
        q = W.f32_to_bf16_bits(rng.standard_normal((B * m, H_q, D), dtype=np.float32) * 0.5)
        logits = W.make_logits(B, m, V, seed=seed + 20 + it)
        tok0, _ = oracle.pmtp_accept(logits, np.zeros((B, m), np.int32))
        drafts = W.mix_drafts(tok0, V, 0.6, seed=seed + 30 + it)
        if it == iters - 1:  # the last step emits fork tokens on the layout branches
            for b in (0, 3):
                logits[b, 0, :] = W.f32_to_bf16_bits(np.full(V, -1.0, np.float32))
                logits[b, 0, FORK] = W.f32_to_bf16_bits(np.array([5.0], np.float32))[0]
                drafts[b, 0] = FORK
        inp = dataclasses.replace(base, q=q, k_cache=st.k_cache, v_cache=st.v_cache,
                                  page_table=st.page_table, branch_len=st.branch_len,
                                  num_pages=st.k_cache.shape[0], max_pages=st.page_table.shape[1])
        d = hpd.DeviceInputs(
            q=bits(q).view(torch.bfloat16), prefix_k=prefix_k, prefix_v=prefix_v,
            prefix_cu=i32(base.prefix_cu), branch_cu=i32(base.branch_cu), branch_prefix_len=None,
            k_cache=kv.k_cache.view(torch.bfloat16), v_cache=kv.v_cache.view(torch.bfloat16),
            page_table=kv.page_table, branch_len=kv.branch_len, n_docs=base.n_docs, B=B, m=m,
            H_q=H_q, H_kv=H_kv, D=D, num_pages=inp.num_pages, max_pages=inp.max_pages,
            prefix_tokens=base.prefix_tokens, max_prefix_len=base.max_prefix_len, scale=0.0)
        op = hpd.BranchAttn(d)
        lg = bits(logits).view(torch.bfloat16)
        out, lse = op.step(lg, i32(drafts), tok, acc)
        torch.cuda.synchronize()
        assert op.errors() == 0 and kv.errors() == 0
        ref_out, ref_lse = oracle.branch_attn(inp)
        assert np.max(np.abs(out.float().cpu().numpy() - ref_out.reshape(out.shape))) <= 1e-2
        fin = ~np.isneginf(ref_lse)
        got_lse = lse.cpu().numpy()
        assert np.array_equal(np.isneginf(got_lse), ~fin)
        assert np.max(np.abs(got_lse[fin] - ref_lse.reshape(got_lse.shape)[fin])) <= 1e-3
        ref_tok, ref_acc = oracle.pmtp_accept(logits, drafts)
        np.testing.assert_array_equal(tok.cpu().numpy(), ref_tok)
        np.testing.assert_array_equal(acc.cpu().numpy(), ref_acc)
        # verification: keep the accepted rows
        st, e = K.rollback(st, ref_acc, m)
        assert e == 0
        kv.rollback(acc)
        torch.cuda.synchronize()
        assert kv.errors() == 0
        np.testing.assert_array_equal(kv.branch_len.cpu().numpy(), st.branch_len)
        np.testing.assert_array_equal(kv.page_table.cpu().numpy(), st.page_table)
        assert int(kv.free_top.item()) == st.top
        np.testing.assert_array_equal(kv.k_cache.cpu().numpy().view(np.uint16), st.k_cache)
        np.testing.assert_array_equal(kv.v_cache.cpu().numpy().view(np.uint16), st.v_cache)
    # fork detection on the last step's emitted tokens: each layout branch
    # (the first of each page) spawned a child at its first emitted token
    is_layout = np.zeros(B, np.int32)
    is_layout[[0, 3]] = 1
    layout_pos = np.maximum(np.repeat(np.diff(base.prefix_cu), np.diff(base.branch_cu)) - m, 0)
    cap = B * (m + 1)
    ref, err = F.fork_children(ref_tok, ref_acc, is_layout, layout_pos, FORK, base.branch_cu, None,
                               st.branch_len, st.page_table, cap)
    assert err == 0 and ref["new_B"] > B
    new = hpd.fork_children(tok, acc, i32(is_layout), i32(layout_pos), FORK, i32(base.branch_cu),
                            None, kv.branch_len, kv.page_table, cap)
    torch.cuda.synchronize()
    assert int(new["workspace"][:4].view(torch.int32).item()) == 0
    nb = ref["new_B"]
    assert int(new["new_B"][0].item()) == nb
    np.testing.assert_array_equal(new["branch_cu"].cpu().numpy(), ref["branch_cu"])
    for k in ("parent", "branch_len", "branch_prefix_len", "page_table"):
        np.testing.assert_array_equal(new[k].cpu().numpy()[:nb], ref[k])
