"""hpd_branch_attn_noalloc: the attention step for callers that cannot
allocate device memory (a plugin whose host engine owns every allocation and
hands it only inputs and outputs, or a path where cudaMalloc is not
allowed).  It keeps its scratch in libhpd's own fixed-size device array
instead of a caller workspace.

These tests call it through the C ABI and check that, on two calls in a row
(the array keeps the previous call's contents), its output matches the
workspace entry point within the parity tolerances, and that a shape needing
more scratch than the array holds is refused.  The file name makes pytest
collect it last.
"""
import numpy as np
import pytest

from paper_2607_18839_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

OUT_TOL = 1e-2
LSE_TOL = 1e-3


@pytest.fixture(scope="module")
def H():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_18839_gb300 import build, hpd
    build.build()
    hpd.load()
    return hpd


def _close(a_out, a_lse, b_out, b_lse):
    assert float((a_out.float() - b_out.float()).abs().max()) <= OUT_TOL
    fin = torch.isfinite(b_lse)
    assert torch.equal(torch.isfinite(a_lse), fin)
    if bool(fin.any()):
        assert float((a_lse[fin] - b_lse[fin]).abs().max()) <= LSE_TOL


@pytest.mark.parametrize("name", ["c2", "multi_page"])
def test_noalloc_matches_workspace_entry_point_on_two_calls(H, name):
    if name == "c2":
        inp = W.make_config("c2")
    else:
        inp = W.build_inputs([300, 0, 77], [3, 2, 4], [0, 5, 16, 1, 40, 2, 31, 32, 200], 4, 16, 2,
                             128, seed=41, extra_pages=3)
    d = H.DeviceInputs.from_host(inp)
    ref = H.BranchAttn(d)
    ref_out, ref_lse = (t.clone() for t in ref())

    out = torch.empty_like(ref_out)
    lse = torch.empty_like(ref_lse)
    args = H.make_args(d, out, lse)  # no workspace: the entry point brings its own
    assert H.hpd_branch_attn_workspace_size(args) <= H.NOALLOC_WORKSPACE_BYTES
    stream = torch.cuda.current_stream()
    for _ in range(2):
        out.fill_(float("nan"))
        lse.fill_(float("nan"))
        H.hpd_branch_attn_noalloc(args, int(stream.cuda_stream) or None)
        torch.cuda.synchronize()
        _close(out, lse, ref_out, ref_lse)


def test_noalloc_refuses_shapes_beyond_its_scratch(H):
    inp = W.make_config("c4")
    args = H.hpd_branch_attn_args()
    for k, v in dict(n_docs=inp.n_docs, B=inp.B, m=inp.m, H_q=inp.H_q, H_kv=inp.H_kv, D=inp.D,
                     num_pages=inp.num_pages, max_pages_per_branch=inp.max_pages,
                     prefix_tokens=inp.prefix_tokens).items():
        setattr(args, k, v)
    # valid (small) device buffers: every argument check passes, so the size
    # is what is refused, before anything is enqueued
    buf = torch.zeros(4096, dtype=torch.uint8, device="cuda")
    for f in ("q", "prefix_k", "prefix_v", "prefix_cu", "branch_cu", "k_cache", "v_cache",
              "page_table", "branch_len", "out", "lse"):
        setattr(args, f, buf.data_ptr())
    assert H.hpd_branch_attn_workspace_size(args) > H.NOALLOC_WORKSPACE_BYTES
    with pytest.raises(H.HpdError) as e:
        H.hpd_branch_attn_noalloc(args, None)
    assert e.value.status == 3  # HPD_ERR_WORKSPACE, nothing enqueued
