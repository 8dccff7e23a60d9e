"""hpd_decode_step: the attention and the greedy acceptance as one step.

The acceptance reads only the logits and the drafts, so the library may run
it beside the attention (on a second stream it forks from and joins to the
caller's stream) when the attention kernel leaves SMs idle.  Whatever it
chooses, the step must give exactly the results of the two calls made in
order, eagerly and inside a captured CUDA graph, and match the oracle.
"""
import numpy as np
import pytest

import oracle
from paper_2607_18839_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

V = 32000


@pytest.fixture(scope="module")
def hpd():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_18839_gb300 import build, hpd as H
    build.build()
    H.load()
    return H


def step_inputs(name, seed):
    inp = W.make_config(name)
    logits = W.make_logits(inp.B, inp.m, V, seed)
    ref_tok0, _ = oracle.pmtp_accept(logits, np.zeros((inp.B, inp.m), np.int32))
    drafts = W.mix_drafts(ref_tok0, V, 0.7, seed=seed + 1)
    return inp, logits, drafts


def to_dev(H, logits, drafts):
    lg = torch.from_numpy(logits.view(np.int16)).cuda().view(torch.bfloat16)
    dr = torch.from_numpy(drafts).cuda()
    return lg, dr


def results(op, tok, acc):
    torch.cuda.synchronize()
    return (op.out.view(torch.int16).cpu().numpy(), op.lse.cpu().numpy(),
            tok.cpu().numpy(), acc.cpu().numpy())


def separate_calls(H, inp, lg, dr):
    op = H.BranchAttn(H.DeviceInputs.from_host(inp))
    tok = torch.empty((inp.B, inp.m), dtype=torch.int32, device="cuda")
    acc = torch.empty((inp.B,), dtype=torch.int32, device="cuda")
    op()
    H.hpd_pmtp_accept(lg.data_ptr(), dr.data_ptr(), inp.B, inp.m, V, tok.data_ptr(),
                      acc.data_ptr(), H._stream_handle(None))
    return results(op, tok, acc)


def assert_same(a, b):
    for x, y, what in zip(a, b, ("out", "lse", "tokens", "accepted_len")):
        assert np.array_equal(x, y, equal_nan=(what == "lse")), what


@pytest.mark.parametrize("name", ["c2", "c3", "c4", "c5"])
def test_step_equals_the_two_calls_bitwise(hpd, name):
    inp, logits, drafts = step_inputs(name, seed=500)
    lg, dr = to_dev(hpd, logits, drafts)
    ref = separate_calls(hpd, inp, lg, dr)
    op = hpd.BranchAttn(hpd.DeviceInputs.from_host(inp))
    tok = torch.full((inp.B, inp.m), -7, dtype=torch.int32, device="cuda")
    acc = torch.full((inp.B,), -7, dtype=torch.int32, device="cuda")
    for _ in range(2):
        op.step(lg, dr, tok, acc)
    got = results(op, tok, acc)
    assert op.errors() == 0
    assert_same(got, ref)


def test_step_matches_the_oracle(hpd):
    inp, logits, drafts = step_inputs("c2", seed=510)
    lg, dr = to_dev(hpd, logits, drafts)
    op = hpd.BranchAttn(hpd.DeviceInputs.from_host(inp))
    tok = torch.empty((inp.B, inp.m), dtype=torch.int32, device="cuda")
    acc = torch.empty((inp.B,), dtype=torch.int32, device="cuda")
    op.step(lg, dr, tok, acc)
    _, lse, tok_np, acc_np = results(op, tok, acc)
    out = op.out.float().cpu().numpy()
    ref_out, ref_lse = oracle.branch_attn(inp)
    assert np.max(np.abs(out - ref_out.reshape(out.shape))) <= 1e-2
    fin = ~np.isneginf(ref_lse)
    assert np.array_equal(np.isneginf(lse), ~fin)
    assert np.max(np.abs(lse[fin] - ref_lse.reshape(lse.shape)[fin])) <= 1e-3
    ref_tok, ref_acc = oracle.pmtp_accept(logits, drafts)
    np.testing.assert_array_equal(tok_np, ref_tok)
    np.testing.assert_array_equal(acc_np, ref_acc)


def test_concurrency_plan(hpd):
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    # beside the attention when there are fewer than two work units per SM:
    # c2 60 units, c5 264 units, c4 832 units (row tiles + one per page, x KV heads x splits)
    for name, units in (("c2", 60), ("c5", 264), ("c4", 832)):
        args = hpd.make_args(hpd.DeviceInputs.from_host(W.make_config(name)))
        assert hpd.hpd_decode_step_concurrent(args) == (1 if units < 2 * sms else 0), name


@pytest.mark.parametrize("name", ["c2", "c4"])
def test_step_inside_graph_capture(hpd, name):
    inp, logits, drafts = step_inputs(name, seed=520)
    lg, dr = to_dev(hpd, logits, drafts)
    ref = separate_calls(hpd, inp, lg, dr)
    op = hpd.BranchAttn(hpd.DeviceInputs.from_host(inp))
    tok = torch.full((inp.B, inp.m), -7, dtype=torch.int32, device="cuda")
    acc = torch.full((inp.B,), -7, dtype=torch.int32, device="cuda")
    s = torch.cuda.Stream()
    op.step(lg, dr, tok, acc, stream=s)  # eager first call (creates the second stream)
    s.synchronize()
    tok.fill_(-7)
    acc.fill_(-7)
    op.out.zero_()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        for _ in range(3):
            op.step(lg, dr, tok, acc, stream=s)
    g.replay()
    got = results(op, tok, acc)
    assert op.errors() == 0
    assert_same(got, ref)


def test_step_refuses_bad_arguments_before_enqueueing(hpd):
    inp, logits, drafts = step_inputs("c2", seed=530)
    lg, dr = to_dev(hpd, logits, drafts)
    op = hpd.BranchAttn(hpd.DeviceInputs.from_host(inp))
    tok = torch.empty((inp.B, inp.m), dtype=torch.int32, device="cuda")
    acc = torch.empty((inp.B,), dtype=torch.int32, device="cuda")
    op.out.fill_(3.0)
    torch.cuda.synchronize()
    lib = hpd.load()
    h = hpd._stream_handle(None)
    # no drafts, then a vocabulary of 0: refused, and the attention did not run
    assert lib.hpd_decode_step(hpd.ctypes.byref(op.args), lg.data_ptr(), None, V,
                               tok.data_ptr(), acc.data_ptr(), h) == 1
    assert lib.hpd_decode_step(hpd.ctypes.byref(op.args), lg.data_ptr(), dr.data_ptr(), 0,
                               tok.data_ptr(), acc.data_ptr(), h) == 1
    torch.cuda.synchronize()
    assert bool((op.out.float() == 3.0).all())


def special_logits(B, m, V, seed):
    """Logits with the cases the argmax must get exactly right: ties (the
    lowest index wins), -0 against +0, NaN (never wins), rows of NaN and -inf
    (the first -inf wins), a row of NaN only (token 0), and maxima at the
    last index and around index 8192."""
    rng = np.random.default_rng(seed)
    x = rng.integers(-4, 5, size=(B, m, V)).astype(np.float32)  # many ties
    x[0, 0, :] = 0.0
    x[0, 0, 7::9] = -0.0
    x[0, 1, :] = np.nan
    x[0, 1, 3] = -np.inf
    x[0, 1, 11] = -np.inf
    x[0, 2, :] = np.nan                      # all NaN -> token 0
    x[1, :, 5::13] = np.nan                  # NaN mixed with values
    x[2, 0, :] = -np.inf
    x[3, 0, V - 1] = 100.0
    if V > 8192:
        x[3, 1, 8192] = 100.0
        x[3, 2, 8191] = 100.0
    return W.f32_to_bf16_bits(x)


@pytest.mark.parametrize("name,V_", [("c4", 4096), ("c4", 20001), ("c2", 32000)])
def test_step_acceptance_special_values(hpd, name, V_):
    inp = W.make_config(name)
    logits = special_logits(inp.B, inp.m, V_, seed=V_)
    ref_tok0, _ = oracle.pmtp_accept(logits, np.zeros((inp.B, inp.m), np.int32))
    drafts = W.mix_drafts(ref_tok0, V_, 0.7, seed=V_ + 1)
    ref_tok, ref_acc = oracle.pmtp_accept(logits, drafts)
    assert ref_tok[0, 2] == 0 and ref_tok[0, 1] == 3 and ref_tok[2, 0] == 0
    lg = torch.from_numpy(logits.view(np.int16)).cuda().view(torch.bfloat16)
    dr = torch.from_numpy(drafts).cuda()
    op = hpd.BranchAttn(hpd.DeviceInputs.from_host(inp))
    tok = torch.full((inp.B, inp.m), -7, dtype=torch.int32, device="cuda")
    acc = torch.full((inp.B,), -7, dtype=torch.int32, device="cuda")
    op.step(lg, dr, tok, acc)
    torch.cuda.synchronize()
    assert op.errors() == 0
    np.testing.assert_array_equal(tok.cpu().numpy(), ref_tok)
    np.testing.assert_array_equal(acc.cpu().numpy(), ref_acc)
