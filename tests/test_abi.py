"""The C-ABI library builds for sm_103a, loads, exports every entry point that
include/hpd.h declares, and rejects bad host arguments before touching the
GPU.  No compute call is made here, so these run without a GPU."""
import ctypes
import os
import re

import numpy as np
import pytest

from paper_2607_18839_gb300 import build as B
from paper_2607_18839_gb300 import hpd

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "hpd.h")


@pytest.fixture(scope="module")
def lib():
    B.build()
    return hpd.load()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(hpd_[a-z0-9_]+)\s*\(", text)))


def test_every_declared_entry_point_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 8
    for n in names:
        assert hasattr(lib, n), f"{n} declared in include/hpd.h but not exported"
    assert set(names) == set(hpd.EXPORTS)


def test_version_and_status_strings(lib):
    assert hpd.hpd_version() >= 100
    assert hpd.hpd_status_string(0) == "ok"
    assert "workspace" in hpd.hpd_status_string(3)


def test_struct_layout_matches_c():
    # 10 pointers, 10 ints, a float, 3 pointers, a size_t, a pointer and an
    # int padded to 8 (x86_64 / aarch64)
    assert ctypes.sizeof(hpd.hpd_branch_attn_args) == 80 + 40 + 8 + 24 + 8 + 8 + 8
    assert hpd.hpd_branch_attn_args.out.offset == 128
    assert hpd.hpd_branch_attn_args.prefix_page_table.offset == 160


def _args(**kw):
    a = hpd.hpd_branch_attn_args()
    base = dict(n_docs=1, B=4, m=4, H_q=16, H_kv=2, D=128, num_pages=10,
                max_pages_per_branch=4, prefix_tokens=100, max_prefix_len=0, scale=0.0)
    base.update(kw)
    for k, v in base.items():
        setattr(a, k, v)
    return a


def test_workspace_size_rejects_bad_scalars(lib):
    assert hpd.hpd_branch_attn_workspace_size(_args()) > 0
    for bad in (dict(D=96), dict(H_q=15), dict(m=0), dict(m=17), dict(B=0), dict(n_docs=0),
                dict(H_q=64, H_kv=2), dict(num_pages=0), dict(max_pages_per_branch=0),
                dict(scale=float("nan")), dict(prefix_page_table=4096, max_prefix_pages=0)):
        assert hpd.hpd_branch_attn_workspace_size(_args(**bad)) == 0, bad


def test_workspace_size_grows_with_rows(lib):
    a = hpd.hpd_branch_attn_workspace_size(_args(B=4))
    b = hpd.hpd_branch_attn_workspace_size(_args(B=64))
    assert b > a > 0


def test_branch_attn_rejects_bad_arguments_before_launch(lib):
    # null device pointers are refused on the host: nothing is launched
    with pytest.raises(hpd.HpdError) as e:
        hpd.hpd_branch_attn(_args(), None)
    assert e.value.status == 1
    with pytest.raises(hpd.HpdError) as e:
        hpd.hpd_branch_attn(_args(D=80), None)
    assert e.value.status == 2


def test_accept_rejects_bad_arguments_before_launch(lib):
    with pytest.raises(hpd.HpdError) as e:
        hpd.hpd_pmtp_accept(None, None, 4, 4, 100, None, None, None)
    assert e.value.status == 1
    with pytest.raises(hpd.HpdError) as e:
        hpd.hpd_pmtp_accept(16, 16, 4, 65, 100, 16, 16, None)
    assert e.value.status == 2


def test_decode_step_rejects_bad_arguments_before_launch(lib):
    # the attention's arguments are checked first, then the acceptance's;
    # either refusal returns before anything reaches a device
    with pytest.raises(hpd.HpdError) as e:
        hpd.hpd_decode_step(_args(), 16, 16, 100, 16, 16, None)
    assert e.value.status == 1
    assert hpd.hpd_decode_step_concurrent(_args(D=80)) == -1


def test_struct_layouts_match_the_header(tmp_path):
    """sizeof / offsetof of the C structs, compiled from include/hpd.h, equal
    the ctypes mirrors of the binding."""
    import shutil
    import subprocess
    if shutil.which("gcc") is None:
        pytest.skip("no gcc")
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    src = tmp_path / "layout.c"
    src.write_text(
        '#include <stdio.h>\n#include <stddef.h>\n#include "hpd.h"\n'
        'int main(void) {\n'
        '  printf("%zu %zu %zu\\n", sizeof(hpd_branch_attn_args), offsetof(hpd_branch_attn_args, out),'
        ' offsetof(hpd_branch_attn_args, workspace_bytes));\n'
        '  printf("%zu %zu\\n", offsetof(hpd_branch_attn_args, prefix_page_table),'
        ' offsetof(hpd_branch_attn_args, max_prefix_pages));\n'
        '  printf("%zu %zu %zu\\n", sizeof(hpd_kv_args), offsetof(hpd_kv_args, workspace),'
        ' offsetof(hpd_kv_args, max_pages));\n'
        '  printf("%zu %zu %zu\\n", sizeof(hpd_fork_args), offsetof(hpd_fork_args, fork_token),'
        ' offsetof(hpd_fork_args, cap));\n'
        '  return 0;\n}\n')
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-I", os.path.join(root, "include"), str(src), "-o", str(exe)], check=True)
    got = [list(map(int, l.split())) for l in subprocess.run([str(exe)], capture_output=True,
                                                              text=True, check=True).stdout.split("\n") if l]
    A, K, F = hpd.hpd_branch_attn_args, hpd.hpd_kv_args, hpd.hpd_fork_args
    assert got[0] == [ctypes.sizeof(A), A.out.offset, A.workspace_bytes.offset]
    assert got[1] == [A.prefix_page_table.offset, A.max_prefix_pages.offset]
    assert got[2] == [ctypes.sizeof(K), K.workspace.offset, K.max_pages.offset]
    assert got[3] == [ctypes.sizeof(F), F.fork_token.offset, F.cap.offset]


def test_noalloc_limit_matches_the_header(tmp_path):
    """The binding's NOALLOC_WORKSPACE_BYTES is the header macro's value."""
    import shutil
    import subprocess
    if shutil.which("gcc") is None:
        pytest.skip("no gcc")
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    src = tmp_path / "limit.c"
    src.write_text('#include <stdio.h>\n#include "hpd.h"\n'
                   'int main(void) { printf("%llu\\n", '
                   '(unsigned long long)HPD_NOALLOC_WORKSPACE_BYTES); return 0; }\n')
    exe = tmp_path / "limit"
    subprocess.run(["gcc", "-I", os.path.join(root, "include"), str(src), "-o", str(exe)], check=True)
    got = int(subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout)
    assert got == hpd.NOALLOC_WORKSPACE_BYTES


def test_noalloc_refuses_bad_arguments_before_enqueueing(lib):
    # null pointers and a misaligned output are refused on the host, before
    # the shared scratch array is touched (no GPU needed)
    with pytest.raises(hpd.HpdError) as e:
        hpd.hpd_branch_attn_noalloc(_args(), None)
    assert e.value.status == 1
    a = _args(q=4096, prefix_k=4096, prefix_v=4096, prefix_cu=4096, branch_cu=4096,
              k_cache=4096, v_cache=4096, page_table=4096, branch_len=4096, out=4098)
    with pytest.raises(hpd.HpdError) as e:
        hpd.hpd_branch_attn_noalloc(a, None)
    assert e.value.status == 1


def _workload_args(inp):
    a = hpd.hpd_branch_attn_args()
    for k, v in dict(n_docs=inp.n_docs, B=inp.B, m=inp.m, H_q=inp.H_q, H_kv=inp.H_kv, D=inp.D,
                     num_pages=inp.num_pages, max_pages_per_branch=inp.max_pages,
                     prefix_tokens=inp.prefix_tokens, max_prefix_len=inp.max_prefix_len,
                     scale=inp.scale).items():
        setattr(a, k, v)
    return a


def big_workload():
    """Three times the 32-page preset's pages (96 pages, 24 branches each)."""
    from paper_2607_18839_gb300 import workloads as W
    rng = np.random.default_rng(77)
    P = rng.integers(1024, 3073, size=96)
    s = np.clip(np.round(rng.lognormal(4.5, 0.8, size=96 * 24)), 1, 1024).astype(np.int64)
    return W.build_inputs(P, [24] * 96, s, 8, 16, 2, 128, seed=78, max_pages=65, name="c4x3")


def test_launch_plan_of_the_workloads(lib):
    # host-only planning: which kernels one call launches (no GPU needed)
    from paper_2607_18839_gb300 import workloads as W
    expect = {
        "c1": ["branch_attn_tc"],                        # one wave, no key split
        "c2": ["branch_attn_tc", "merge_splits"],        # few tiles: keys split, then merged
        "c4": ["branch_attn_tc"],                        # the order pass would not pay
        "c5": ["branch_attn_tc"],
    }
    for name, kernels in expect.items():
        a = _workload_args(W.make_config(name))
        n = hpd.hpd_branch_attn_launches(a)
        got = [hpd.hpd_branch_attn_kernel_name(a, k) for k in range(n)]
        assert got == kernels, (name, got)
        assert hpd.hpd_branch_attn_kernel_name(a, n) is None
    # a large step (96 pages) orders its work units longest first
    assert [hpd.hpd_branch_attn_kernel_name(_workload_args(big_workload()), k) for k in range(2)] == [
        "unit_order", "branch_attn_tc"]
    # head ratios that do not divide 128 take the warp-MMA stages
    g3 = W.build_inputs([200], [3], [4, 0, 33], 3, 6, 2, 128, seed=1)
    a = _workload_args(g3)
    assert [hpd.hpd_branch_attn_kernel_name(a, k) for k in range(2)] == ["prefix_stage",
                                                                        "suffix_merge"]
    # the unit order lives in the workspace: it grows with the units
    assert hpd.hpd_branch_attn_workspace_size(_workload_args(W.make_config("c4"))) > 0
