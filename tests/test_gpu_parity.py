"""Parity of the CUDA path (through the C ABI) with the fp64 oracle.

Tolerances (fixed for the branch-decode step): attention output max abs error
<= 1e-2 (bf16 output, fp32 accumulation), LSE within 1e-3, -inf LSE exactly
where the oracle has no visible key; accepted lengths and tokens bit-exact.
Small workloads and the full-size presets c3, c4 and c5 are compared element
by element on every row; quicker checks compare a sample of branches chosen
to include the extreme suffix lengths and every page boundary kind.
"""
import numpy as np
import pytest

import oracle
from paper_2607_18839_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

OUT_TOL = 1e-2
LSE_TOL = 1e-3


@pytest.fixture(scope="module")
def hpd():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_18839_gb300 import build, hpd as H
    build.build()
    H.load()
    return H


def run_gpu(H, inp):
    d = H.DeviceInputs.from_host(inp)
    op = H.BranchAttn(d)
    out, lse = op()
    torch.cuda.synchronize()
    err = op.errors()
    return out.float().cpu().numpy(), lse.cpu().numpy(), err


def compare(inp, out, lse, ref_out, ref_lse, rows=None):
    if rows is not None:
        out, lse, ref_out, ref_lse = out[rows], lse[rows], ref_out[rows], ref_lse[rows]
    neg = np.isneginf(ref_lse)
    assert np.array_equal(np.isneginf(lse), neg), "-inf LSE pattern differs"
    assert np.all(np.isfinite(lse[~neg]))
    if (~neg).any():
        lerr = np.max(np.abs(lse[~neg] - ref_lse[~neg]))
        assert lerr <= LSE_TOL, f"lse err {lerr}"
    oerr = np.max(np.abs(out - ref_out))
    assert oerr <= OUT_TOL, f"out err {oerr}"
    return oerr


def branch_rows(inp, branches):
    branches = np.asarray(branches)
    return (branches[:, None] * inp.m + np.arange(inp.m)[None, :]).reshape(-1)


SMALL = {
    "c1": lambda: W.make_config("c1"),
    "c2": lambda: W.make_config("c2"),
    # several pages, ragged row tiles, private lengths 0 / < m / page multiples
    "multi_page_ragged": lambda: W.build_inputs(
        [300, 0, 77, 129], [3, 2, 1, 5], [0, 5, 16, 1, 40, 2, 31, 32, 48, 200, 3],
        4, 16, 2, 128, seed=31, extra_pages=7),
    "fork_prefix_lengths": lambda: W.build_inputs(
        [500, 200], [4, 3], [10, 20, 30, 40, 0, 1, 2], 3, 8, 4, 128, seed=32,
        branch_prefix_len=[500, 0, 1, 250, 200, 63, 64]),
    "d64_g1": lambda: W.build_inputs([333], [5], [1, 17, 33, 65, 129], 2, 4, 4, 64, seed=33),
    "g16_m16": lambda: W.build_inputs([100, 260], [2, 2], [0, 15, 16, 300], 16, 16, 1, 128,
                                      seed=34),
    "m1_empty_suffix": lambda: W.build_inputs([1152], [16], [0] * 16, 1, 16, 2, 128, seed=35),
    "no_prefix_at_all": lambda: W.build_inputs([0], [3], [0, 4, 50], 4, 8, 2, 128, seed=36),
    "long_suffix_splits": lambda: W.build_inputs([64], [2], [2047, 1500], 4, 32, 8, 128, seed=37,
                                                 max_pages=129),
    "custom_scale": lambda: W.build_inputs([90], [2], [7, 9], 2, 4, 2, 64, seed=38, scale=0.3),
    # G = 3 and G = 5 do not divide 128: these take the warp-MMA prefix kernel
    "g3_warp_mma_prefix": lambda: W.build_inputs([200, 50], [3, 2], [4, 0, 33, 17, 64], 3, 6, 2,
                                                 128, seed=42, branch_prefix_len=[200, 7, 150, 50, 0]),
    "g5_d64_warp_mma_prefix": lambda: W.build_inputs([129], [4], [1, 2, 3, 100], 2, 10, 2, 64,
                                                     seed=43),
    # m G = 64: row tiles of two branches, whose private pages fill one half of
    # each suffix block each (lengths L = s + m of 8, 64, 65, 128, 308 keys:
    # empty halves, segment ends, several blocks), plus one-branch tiles
    "two_branch_tiles": lambda: W.build_inputs(
        [700, 130, 0], [5, 2, 3], [0, 1, 56, 57, 120, 200, 8, 300, 63, 64], 8, 16, 2, 128,
        seed=49),
    "two_branch_tiles_d64_fork": lambda: W.build_inputs(
        [400, 90], [4, 2], [3, 250, 60, 0, 17, 129], 4, 16, 1, 64, seed=50,
        branch_prefix_len=[400, 0, 128, 399, 90, 1]),
    # many pages with one branch each, long prefixes split across CTAs
    "many_pages_split_prefix": lambda: W.build_inputs([1000 + 37 * i for i in range(12)], [1] * 12,
                                                      [5 * i for i in range(12)], 4, 16, 2, 128,
                                                      seed=44),
}


@pytest.mark.parametrize("name", list(SMALL))
def test_parity_small_elementwise(hpd, name):
    inp = SMALL[name]()
    ref_out, ref_lse = oracle.branch_attn(inp)
    out, lse, err = run_gpu(hpd, inp)
    assert err == 0
    compare(inp, out, lse, ref_out, ref_lse)


def sample_branches(inp, k=6):
    s = inp.branch_len
    picks = {0, inp.B - 1, int(np.argmax(s)), int(np.argmin(s))}
    for d in (0, inp.n_docs - 1):
        picks.update({int(inp.branch_cu[d]), int(inp.branch_cu[d + 1]) - 1})
    rng = np.random.default_rng(5)
    picks.update(rng.choice(inp.B, size=min(k, inp.B), replace=False).tolist())
    return sorted(b for b in picks if 0 <= b < inp.B)


@pytest.mark.parametrize("name", ["c3", "c4", "c5"])
def test_parity_full_size_sampled_branches(hpd, name):
    # quick check on a sample of branches (the every-row tests follow)
    inp = W.make_config(name)
    sel = np.array(sample_branches(inp), dtype=np.int32)
    ref_out, ref_lse = oracle.branch_attn(inp, branch_sel=sel)
    out, lse, err = run_gpu(hpd, inp)
    assert err == 0
    compare(inp, out, lse, ref_out, ref_lse, rows=branch_rows(inp, sel))


_FULL_ORACLE = {}


def full_oracle(name):
    """The oracle over every row of a preset (computed once per session)."""
    if name not in _FULL_ORACLE:
        _FULL_ORACLE[name] = oracle.branch_attn(W.make_config(name))
    return _FULL_ORACLE[name]


@pytest.mark.parametrize("name", ["c4", "c5"])
def test_parity_full_size_every_row(hpd, name):
    # every row of every row tile, KV head and split of the preset
    inp = W.make_config(name)
    ref_out, ref_lse = full_oracle(name)
    out, lse, err = run_gpu(hpd, inp)
    assert err == 0
    compare(inp, out, lse, ref_out, ref_lse)


def test_unit_with_more_suffix_pages_than_the_shared_table(hpd):
    # G = 1, m = 1: one 128-row tile holds 128 branches whose private
    # histories pack ~3,300 pages, past the 2,048 page ids a unit keeps in
    # shared memory, so the later pages are looked up again in the table
    rng = np.random.default_rng(48)
    s = rng.integers(20 * 16, 32 * 16 + 1, size=128)
    inp = W.build_inputs([50], [128], s, 1, 1, 1, 64, seed=48, max_pages=33)
    assert int(np.ceil(inp.branch_len / W.PAGE).sum()) > 2048
    ref_out, ref_lse = oracle.branch_attn(inp)
    out, lse, err = run_gpu(hpd, inp)
    assert err == 0
    compare(inp, out, lse, ref_out, ref_lse)


# ----------------------------------------------------------- paged prefix --

@pytest.mark.parametrize("name", list(SMALL))
def test_paged_prefix_small_elementwise(hpd, name):
    # the prefix read through the page pool (contiguous buffers not passed)
    inp = W.page_the_prefix(SMALL[name](), seed=90, extra_pages=3)
    ref_out, ref_lse = oracle.branch_attn(inp)
    out, lse, err = run_gpu(hpd, inp)
    assert err == 0
    compare(inp, out, lse, ref_out, ref_lse)


@pytest.mark.parametrize("runs", [False, True])
@pytest.mark.parametrize("name", ["c2", "c4", "g3_warp_mma_prefix", "many_pages_split_prefix"])
def test_paged_prefix_equals_contiguous_bitwise(hpd, name, runs):
    # same keys in the same blocks: the paged and contiguous layouts give
    # identical bits (masked slots weigh exactly zero in both); with runs the
    # prefix pages are consecutive in the pool and load as 8-page boxes
    base = SMALL[name]() if name in SMALL else W.make_config(name)
    o1, l1, e1 = run_gpu(hpd, base)
    o2, l2, e2 = run_gpu(hpd, W.page_the_prefix(base, seed=91, runs=runs))
    assert e1 == e2 == 0
    np.testing.assert_array_equal(o1, o2)
    np.testing.assert_array_equal(l1, l2)


@pytest.mark.parametrize("runs", [False, True])
@pytest.mark.parametrize("name", ["c3", "c4", "c5"])
def test_paged_prefix_full_size_sampled_branches(hpd, name, runs):
    inp = W.page_the_prefix(W.make_config(name), seed=92, runs=runs)
    sel = np.array(sample_branches(inp), dtype=np.int32)
    ref_out, ref_lse = oracle.branch_attn(inp, branch_sel=sel)
    out, lse, err = run_gpu(hpd, inp)
    assert err == 0
    compare(inp, out, lse, ref_out, ref_lse, rows=branch_rows(inp, sel))


@pytest.mark.parametrize("runs", [False, True])
@pytest.mark.parametrize("name", ["c4", "c5"])
def test_paged_prefix_full_size_every_row(hpd, name, runs):
    # the paged layout holds the same keys as the contiguous one (pinned on
    # the CPU: the oracle's paged mode equals its contiguous mode), so every
    # row is compared with the oracle of the contiguous preset
    inp = W.page_the_prefix(W.make_config(name), seed=92, runs=runs)
    ref_out, ref_lse = full_oracle(name)
    out, lse, err = run_gpu(hpd, inp)
    assert err == 0
    compare(inp, out, lse, ref_out, ref_lse)


def _defragment(inp):
    """The same workload with each branch's private pages made consecutive
    pool pages (in branch order), the unused pages after them."""
    used = [int(p) for b in range(inp.B)
            for p in inp.page_table[b, :(int(inp.branch_len[b]) + W.PAGE - 1) // W.PAGE]]
    rest = [p for p in range(inp.num_pages) if p not in set(used)]
    order = np.array(used + rest, np.int64)        # new id -> old id
    new_of = np.empty(inp.num_pages, np.int32)
    new_of[order] = np.arange(inp.num_pages, dtype=np.int32)
    out = W.BranchDecodeInputs(**{**inp.__dict__})
    out.k_cache, out.v_cache = inp.k_cache[order], inp.v_cache[order]
    out.page_table = new_of[inp.page_table]
    return out


@pytest.mark.parametrize("name", ["c3", "long_suffix_splits"])
def test_consecutive_private_pages_bitwise(hpd, name):
    # private pages in consecutive pool pages load as 8-page boxes; the
    # result is the same bits as with scattered pages
    base = SMALL[name]() if name in SMALL else W.make_config(name)
    o1, l1, e1 = run_gpu(hpd, base)
    o2, l2, e2 = run_gpu(hpd, _defragment(base))
    assert e1 == e2 == 0
    np.testing.assert_array_equal(o1, o2)
    np.testing.assert_array_equal(l1, l2)


def test_paged_prefix_table_too_narrow_is_flagged(hpd):
    # a prefix page table with fewer columns than the page's prefix needs:
    # the prefix is cut at the table's end and HPD_DEVERR_PREFIX_CU is set
    inp = W.page_the_prefix(W.build_inputs([100], [2], [3, 4], 2, 8, 2, 128, seed=46), seed=94)
    inp.prefix_page_table = np.ascontiguousarray(inp.prefix_page_table[:, :4])  # 64 of 100 tokens
    out, lse, err = run_gpu(hpd, inp)
    assert err & 0x1
    assert np.all(np.isfinite(out)) and np.all(np.isfinite(lse))


def test_paged_prefix_bad_page_id_is_flagged(hpd):
    inp = W.page_the_prefix(W.build_inputs([100], [2], [3, 4], 2, 8, 2, 128, seed=45), seed=93)
    inp.prefix_page_table[0, 1] = inp.num_pages + 5
    out, lse, err = run_gpu(hpd, inp)
    assert err & 0x8
    assert np.all(np.isfinite(out))


def test_parity_large_step_with_ordered_units(hpd):
    # 96 pages: long enough that the work units are ordered longest first
    from test_abi import big_workload
    inp = big_workload()
    d = hpd.DeviceInputs.from_host(inp)
    op = hpd.BranchAttn(d)
    names = [hpd.hpd_branch_attn_kernel_name(op.args, k)
             for k in range(hpd.hpd_branch_attn_launches(op.args))]
    assert names == ["unit_order", "branch_attn_tc"]
    out, lse = op()
    torch.cuda.synchronize()
    assert op.errors() == 0
    ref_out, ref_lse = oracle.branch_attn(inp)  # every row
    compare(inp, out.float().cpu().numpy(), lse.cpu().numpy(), ref_out, ref_lse)


def test_c3_full_oracle_elementwise(hpd):
    inp = W.make_config("c3")
    ref_out, ref_lse = oracle.branch_attn(inp)
    out, lse, _ = run_gpu(hpd, inp)
    compare(inp, out, lse, ref_out, ref_lse)


def test_repeated_calls_are_deterministic(hpd):
    inp = W.make_config("c2")
    d = hpd.DeviceInputs.from_host(inp)
    op = hpd.BranchAttn(d)
    o1 = op()[0].clone()
    o2 = op()[0].clone()
    torch.cuda.synchronize()
    assert torch.equal(o1, o2)


@pytest.mark.parametrize("name", ["c2", "c4"])
def test_marked_call_outside_and_inside_capture(hpd, name):
    """hpd_branch_attn_marked: same results as the plain call, one timed
    interval per kernel, eager and inside a captured graph."""
    inp = W.make_config(name)
    d = hpd.DeviceInputs.from_host(inp)
    op = hpd.BranchAttn(d)
    ref = op()[0].clone()
    n = hpd.hpd_branch_attn_launches(op.args)
    names = [hpd.hpd_branch_attn_kernel_name(op.args, k) for k in range(n)]
    assert "branch_attn_tc" in names and hpd.hpd_branch_attn_kernel_name(op.args, n) is None
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(n + 1)]
    for e in ev:
        e.record()
    torch.cuda.synchronize()
    op.out.zero_()
    op(events=ev)
    torch.cuda.synchronize()
    assert torch.equal(op.out, ref)
    assert all(ev[k].elapsed_time(ev[k + 1]) > 0 for k in range(n))
    g = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        op()  # warm on the capture stream
        s.synchronize()
        with torch.cuda.graph(g, stream=s):
            op(stream=s, events=ev)
    op.out.zero_()
    g.replay()
    torch.cuda.synchronize()
    assert torch.equal(op.out, ref)
    assert ev[0].elapsed_time(ev[n]) > 0


@pytest.mark.parametrize("name", ["c1", "multi_page_ragged", "c2"])
def test_output_only_16_byte_aligned(hpd, name):
    # the ABI asks 16-byte alignment of out; the kernel's 32-byte stores are
    # used only when out allows them
    inp = SMALL[name]()
    d = hpd.DeviceInputs.from_host(inp)
    op = hpd.BranchAttn(d)
    ref = op()[0].clone()
    n = ref.numel()
    big = torch.zeros(n + 8, dtype=torch.bfloat16, device=ref.device)
    out16 = big[8:].view(ref.shape)  # 16 bytes past a 256-byte boundary
    assert out16.data_ptr() % 32 == 16
    args = hpd.make_args(d, out16, op.lse, op.workspace, op.workspace.numel())
    hpd.hpd_branch_attn(args, hpd._stream_handle(None))
    torch.cuda.synchronize()
    assert op.errors() == 0
    assert torch.equal(out16, ref)


def test_out_of_range_device_data_is_clamped_and_flagged(hpd):
    inp = W.build_inputs([40], [2], [20, 30], 2, 8, 2, 64, seed=39)
    inp.page_table[1, 0] = inp.num_pages + 5   # page id out of range
    inp.branch_len[0] = 10_000                   # beyond the page table
    out, lse, err = run_gpu(hpd, inp)
    assert err & 0x8 and err & 0x4
    assert np.all(np.isfinite(out))


# ------------------------------------------------------------- acceptance --

def run_accept(hpd, logits_bits, drafts):
    lg = torch.from_numpy(np.ascontiguousarray(logits_bits).view(np.int16)).cuda().view(torch.bfloat16)
    dr = torch.from_numpy(np.ascontiguousarray(drafts, dtype=np.int32)).cuda()
    tok, acc = hpd.pmtp_accept(lg, dr)
    torch.cuda.synchronize()
    return tok.cpu().numpy(), acc.cpu().numpy()


def test_accept_c5_bit_exact(hpd):
    logits = W.accept_inputs()
    ref_tok0, _ = oracle.pmtp_accept(logits, np.zeros(logits.shape[:2], np.int32))
    drafts = W.mix_drafts(ref_tok0, logits.shape[2], 0.7, seed=77)
    ref_tok, ref_acc = oracle.pmtp_accept(logits, drafts)
    tok, acc = run_accept(hpd, logits, drafts)
    np.testing.assert_array_equal(tok, ref_tok)
    np.testing.assert_array_equal(acc, ref_acc)
    assert 0 < ref_acc.mean() < 4


@pytest.mark.parametrize("V", [1, 7, 8, 9, 4095, 32001])
def test_accept_ragged_vocab_ties_and_nan(hpd, V):
    rng = np.random.default_rng(V)
    B, m = 5, 6
    vals = rng.integers(-3, 4, size=(B, m, V)).astype(np.float32)  # many ties
    vals[0, 0, :] = np.nan
    vals[1, 1, V // 2] = np.nan
    vals[2, 2, :] = -np.inf
    vals[3, 3, :] = -np.inf             # the maximum is -inf, first after a run of NaN
    vals[3, 3, :(V + 2) // 3] = np.nan
    vals[4, 4, :] = np.nan              # a single -inf at the end
    vals[4, 4, V - 1] = -np.inf
    logits = W.f32_to_bf16_bits(vals)
    ref_tok0, _ = oracle.pmtp_accept(logits, np.zeros((B, m), np.int32))
    drafts = W.mix_drafts(ref_tok0, V, 0.8, seed=V + 1)
    ref_tok, ref_acc = oracle.pmtp_accept(logits, drafts)
    tok, acc = run_accept(hpd, logits, drafts)
    np.testing.assert_array_equal(tok, ref_tok)
    np.testing.assert_array_equal(acc, ref_acc)


def test_accept_more_rows_than_the_cluster(hpd):
    # m = 12 > 8 CTAs per cluster: CTAs take two rows each in turn; -inf rows
    # land on a CTA's second row
    rng = np.random.default_rng(12)
    B, m, V = 7, 12, 1000
    vals = rng.integers(-2, 3, size=(B, m, V)).astype(np.float32)
    vals[1, 9, :] = -np.inf
    vals[1, 9, :500] = np.nan
    vals[2, 11, :] = np.nan
    vals[3, 8, :] = -np.inf
    logits = W.f32_to_bf16_bits(vals)
    ref_tok0, _ = oracle.pmtp_accept(logits, np.zeros((B, m), np.int32))
    drafts = W.mix_drafts(ref_tok0, V, 0.9, seed=13)
    ref_tok, ref_acc = oracle.pmtp_accept(logits, drafts)
    tok, acc = run_accept(hpd, logits, drafts)
    np.testing.assert_array_equal(tok, ref_tok)
    np.testing.assert_array_equal(acc, ref_acc)
    assert ref_tok[1, 9] == 500 and ref_tok[3, 8] == 0


def test_accept_misaligned_rows(hpd):
    # V = 33 makes every row start at a different 16-byte phase
    rng = np.random.default_rng(2)
    logits = W.f32_to_bf16_bits(rng.standard_normal((9, 7, 33)).astype(np.float32))
    ref_tok, ref_acc = oracle.pmtp_accept(logits, np.zeros((9, 7), np.int32))
    tok, acc = run_accept(hpd, logits, np.zeros((9, 7), np.int32))
    np.testing.assert_array_equal(tok, ref_tok)
    np.testing.assert_array_equal(acc, ref_acc)
