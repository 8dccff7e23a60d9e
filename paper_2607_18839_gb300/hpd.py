"""Thin ctypes binding of libhpd (include/hpd.h), same entry-point names.

Argument marshalling only: every step of the branch-decode path runs in the
CUDA kernels behind the C ABI.  torch tensors supply device memory and
streams.  There is no fallback: if ``libhpd.so`` is missing, or a call is
made without a CUDA device, the call raises.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass
from typing import Optional

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "libhpd.so")

HPD_OK = 0
STATUS = {0: "HPD_OK", 1: "HPD_ERR_INVALID_ARG", 2: "HPD_ERR_UNSUPPORTED",
          3: "HPD_ERR_WORKSPACE", 4: "HPD_ERR_CUDA", 5: "HPD_ERR_TIMEOUT"}

DEVERR = {0x1: "PREFIX_CU", 0x2: "BRANCH_CU", 0x4: "BRANCH_LEN", 0x8: "PAGE_ID",
          0x10: "FORK_LEN", 0x40: "TIMEOUT"}

# Every entry point declared in include/hpd.h.
EXPORTS = ("hpd_branch_attn_workspace_size", "hpd_workspace_init", "hpd_branch_attn",
           "hpd_branch_attn_launches", "hpd_branch_attn_kernel_name", "hpd_branch_attn_marked",
           "hpd_pmtp_accept", "hpd_decode_step", "hpd_decode_step_concurrent",
           "hpd_read_errors", "hpd_status_string", "hpd_last_cuda_error", "hpd_version",
           "hpd_branch_attn_noalloc", "hpd_wait_selftest", "hpd_kv_append", "hpd_kv_rollback",
           "hpd_fork_children")

# Scratch bytes built into libhpd for hpd_branch_attn_noalloc.
NOALLOC_WORKSPACE_BYTES = 32 << 20


class HpdError(RuntimeError):
    def __init__(self, fn: str, status: int, detail: str = ""):
        self.status = status
        super().__init__(f"{fn} -> {STATUS.get(status, status)}{(': ' + detail) if detail else ''}")


class hpd_branch_attn_args(ctypes.Structure):
    """Mirror of the C struct of the same name."""

    _fields_ = [
        ("q", ctypes.c_void_p), ("prefix_k", ctypes.c_void_p), ("prefix_v", ctypes.c_void_p),
        ("prefix_cu", ctypes.c_void_p), ("branch_cu", ctypes.c_void_p),
        ("branch_prefix_len", ctypes.c_void_p), ("k_cache", ctypes.c_void_p),
        ("v_cache", ctypes.c_void_p), ("page_table", ctypes.c_void_p),
        ("branch_len", ctypes.c_void_p),
        ("n_docs", ctypes.c_int), ("B", ctypes.c_int), ("m", ctypes.c_int),
        ("H_q", ctypes.c_int), ("H_kv", ctypes.c_int), ("D", ctypes.c_int),
        ("num_pages", ctypes.c_int), ("max_pages_per_branch", ctypes.c_int),
        ("prefix_tokens", ctypes.c_int), ("max_prefix_len", ctypes.c_int),
        ("scale", ctypes.c_float),
        ("out", ctypes.c_void_p), ("lse", ctypes.c_void_p),
        ("workspace", ctypes.c_void_p), ("workspace_bytes", ctypes.c_size_t),
        ("prefix_page_table", ctypes.c_void_p), ("max_prefix_pages", ctypes.c_int),
    ]


class hpd_kv_args(ctypes.Structure):
    """Mirror of the C struct of the same name."""

    _fields_ = [
        ("k_new", ctypes.c_void_p), ("v_new", ctypes.c_void_p),
        ("k_cache", ctypes.c_void_p), ("v_cache", ctypes.c_void_p),
        ("page_table", ctypes.c_void_p), ("branch_len", ctypes.c_void_p),
        ("free_pages", ctypes.c_void_p), ("free_top", ctypes.c_void_p),
        ("workspace", ctypes.c_void_p),
        ("B", ctypes.c_int), ("m", ctypes.c_int), ("H_kv", ctypes.c_int), ("D", ctypes.c_int),
        ("num_pages", ctypes.c_int), ("max_pages", ctypes.c_int),
    ]


class hpd_fork_args(ctypes.Structure):
    """Mirror of the C struct of the same name."""

    _fields_ = [(n, ctypes.c_void_p) for n in (
        "out_tokens", "accepted_len", "is_layout", "layout_pos", "branch_cu", "branch_prefix_len",
        "branch_len", "page_table", "new_branch_cu", "new_branch_prefix_len", "new_branch_len",
        "new_page_table", "new_parent", "new_B", "workspace")] + [
        ("workspace_bytes", ctypes.c_size_t), ("fork_token", ctypes.c_int32),
        ("B", ctypes.c_int), ("m", ctypes.c_int), ("n_docs", ctypes.c_int),
        ("max_pages", ctypes.c_int), ("cap", ctypes.c_int)]


_lib = None


def load(path: str = LIB_PATH):
    """Load libhpd.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with "
                           "`python -m paper_2607_18839_gb300.build`")
    lib = ctypes.CDLL(path)
    P, I, S = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t
    lib.hpd_branch_attn_workspace_size.restype = S
    lib.hpd_branch_attn_workspace_size.argtypes = [ctypes.POINTER(hpd_branch_attn_args)]
    lib.hpd_workspace_init.restype = I
    lib.hpd_workspace_init.argtypes = [P, S, P]
    lib.hpd_branch_attn.restype = I
    lib.hpd_branch_attn.argtypes = [ctypes.POINTER(hpd_branch_attn_args), P]
    lib.hpd_branch_attn_launches.restype = I
    lib.hpd_branch_attn_launches.argtypes = [ctypes.POINTER(hpd_branch_attn_args)]
    lib.hpd_branch_attn_kernel_name.restype = ctypes.c_char_p
    lib.hpd_branch_attn_kernel_name.argtypes = [ctypes.POINTER(hpd_branch_attn_args), I]
    lib.hpd_branch_attn_marked.restype = I
    lib.hpd_branch_attn_marked.argtypes = [ctypes.POINTER(hpd_branch_attn_args), P,
                                           ctypes.POINTER(ctypes.c_void_p)]
    lib.hpd_pmtp_accept.restype = I
    lib.hpd_pmtp_accept.argtypes = [P, P, I, I, I, P, P, P]
    lib.hpd_decode_step.restype = I
    lib.hpd_decode_step.argtypes = [ctypes.POINTER(hpd_branch_attn_args), P, P, I, P, P, P]
    lib.hpd_decode_step_concurrent.restype = I
    lib.hpd_decode_step_concurrent.argtypes = [ctypes.POINTER(hpd_branch_attn_args)]
    lib.hpd_read_errors.restype = I
    lib.hpd_read_errors.argtypes = [P, ctypes.POINTER(ctypes.c_uint32), P]
    lib.hpd_status_string.restype = ctypes.c_char_p
    lib.hpd_status_string.argtypes = [I]
    lib.hpd_last_cuda_error.restype = I
    lib.hpd_last_cuda_error.argtypes = []
    lib.hpd_version.restype = I
    lib.hpd_version.argtypes = []
    lib.hpd_branch_attn_noalloc.restype = I
    lib.hpd_branch_attn_noalloc.argtypes = [ctypes.POINTER(hpd_branch_attn_args), P]
    lib.hpd_wait_selftest.restype = I
    lib.hpd_wait_selftest.argtypes = [P, ctypes.c_uint32, P]
    lib.hpd_kv_append.restype = I
    lib.hpd_kv_append.argtypes = [ctypes.POINTER(hpd_kv_args), P]
    lib.hpd_kv_rollback.restype = I
    lib.hpd_kv_rollback.argtypes = [ctypes.POINTER(hpd_kv_args), P, P]
    lib.hpd_fork_children.restype = I
    lib.hpd_fork_children.argtypes = [ctypes.POINTER(hpd_fork_args), P]
    _lib = lib
    return lib


def _check(fn: str, status: int):
    if status != HPD_OK:
        detail = ""
        if status == 4:
            detail = f"cudaError {load().hpd_last_cuda_error()}"
        raise HpdError(fn, status, detail)


def _ptr(t) -> Optional[int]:
    return None if t is None else int(t.data_ptr())


def _stream_handle(stream) -> Optional[int]:
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream) or None


# ------------------------------------------------------------ raw C calls --

def hpd_branch_attn_workspace_size(args: hpd_branch_attn_args) -> int:
    return int(load().hpd_branch_attn_workspace_size(ctypes.byref(args)))


def hpd_workspace_init(workspace_ptr: int, nbytes: int, stream_handle: Optional[int]) -> None:
    _check("hpd_workspace_init", load().hpd_workspace_init(workspace_ptr, nbytes, stream_handle))


def hpd_branch_attn(args: hpd_branch_attn_args, stream_handle: Optional[int]) -> None:
    _check("hpd_branch_attn", load().hpd_branch_attn(ctypes.byref(args), stream_handle))


def hpd_branch_attn_launches(args: hpd_branch_attn_args) -> int:
    return int(load().hpd_branch_attn_launches(ctypes.byref(args)))


def hpd_branch_attn_kernel_name(args: hpd_branch_attn_args, k: int) -> Optional[str]:
    name = load().hpd_branch_attn_kernel_name(ctypes.byref(args), k)
    return None if name is None else name.decode()


def hpd_branch_attn_marked(args: hpd_branch_attn_args, stream_handle, event_handles) -> None:
    """``event_handles``: ints (cudaEvent_t), launches + 1 of them."""
    arr = (ctypes.c_void_p * len(event_handles))(*event_handles)
    _check("hpd_branch_attn_marked", load().hpd_branch_attn_marked(ctypes.byref(args),
                                                                    stream_handle, arr))


def hpd_pmtp_accept(logits_ptr, drafts_ptr, B, m, V, out_tokens_ptr, accepted_len_ptr,
                    stream_handle) -> None:
    _check("hpd_pmtp_accept", load().hpd_pmtp_accept(logits_ptr, drafts_ptr, B, m, V,
                                                     out_tokens_ptr, accepted_len_ptr,
                                                     stream_handle))


def hpd_decode_step(args: hpd_branch_attn_args, logits_ptr, drafts_ptr, V, out_tokens_ptr,
                    accepted_len_ptr, stream_handle) -> None:
    """hpd_branch_attn(args) and hpd_pmtp_accept (B = args.B, m = args.m) as
    one step; the acceptance runs beside the attention when the attention
    leaves SMs idle (see include/hpd.h)."""
    _check("hpd_decode_step", load().hpd_decode_step(ctypes.byref(args), logits_ptr, drafts_ptr,
                                                     V, out_tokens_ptr, accepted_len_ptr,
                                                     stream_handle))


def hpd_decode_step_concurrent(args: hpd_branch_attn_args) -> int:
    return int(load().hpd_decode_step_concurrent(ctypes.byref(args)))


def hpd_read_errors(workspace_ptr: int, stream_handle) -> int:
    flags = ctypes.c_uint32(0)
    _check("hpd_read_errors", load().hpd_read_errors(workspace_ptr, ctypes.byref(flags),
                                                      stream_handle))
    return int(flags.value)


def hpd_wait_selftest(workspace_ptr: int, limit_us: int, stream_handle) -> None:
    _check("hpd_wait_selftest", load().hpd_wait_selftest(workspace_ptr, limit_us, stream_handle))


def hpd_kv_append(args: hpd_kv_args, stream_handle) -> None:
    _check("hpd_kv_append", load().hpd_kv_append(ctypes.byref(args), stream_handle))


def hpd_kv_rollback(args: hpd_kv_args, accepted_len_ptr: int, stream_handle) -> None:
    _check("hpd_kv_rollback", load().hpd_kv_rollback(ctypes.byref(args), accepted_len_ptr,
                                                      stream_handle))


def hpd_branch_attn_noalloc(args: hpd_branch_attn_args, stream_handle: Optional[int]) -> None:
    """The step with libhpd's built-in scratch array instead of a workspace
    (for callers that cannot allocate; see include/hpd.h)."""
    _check("hpd_branch_attn_noalloc", load().hpd_branch_attn_noalloc(ctypes.byref(args),
                                                                      stream_handle))


def hpd_status_string(status: int) -> str:
    return load().hpd_status_string(status).decode()


def hpd_version() -> int:
    return int(load().hpd_version())


# ------------------------------------------------------- torch conveniences --

@dataclass
class DeviceInputs:
    """Device copies of one workload's inputs (torch tensors)."""

    q: "object"
    prefix_k: "object"
    prefix_v: "object"
    prefix_cu: "object"
    branch_cu: "object"
    branch_prefix_len: "object"
    k_cache: "object"
    v_cache: "object"
    page_table: "object"
    branch_len: "object"
    n_docs: int
    B: int
    m: int
    H_q: int
    H_kv: int
    D: int
    num_pages: int
    max_pages: int
    prefix_tokens: int
    max_prefix_len: int
    scale: float
    prefix_page_table: "object" = None  # paged prefix: int32 [n_docs, max_prefix_pages]
    max_prefix_pages: int = 0

    @staticmethod
    def from_host(inp, device="cuda", non_blocking=False) -> "DeviceInputs":
        """Copy a ``workloads.BranchDecodeInputs`` to the device (with a paged
        prefix, the contiguous prefix buffers are not copied)."""
        import numpy as np
        import torch

        def bf(a):
            if a is None:
                return None
            t = torch.from_numpy(np.ascontiguousarray(a).view(np.int16))
            return t.to(device, non_blocking=non_blocking).view(torch.bfloat16)

        def i32(a):
            return None if a is None else torch.from_numpy(
                np.ascontiguousarray(a, dtype=np.int32)).to(device, non_blocking=non_blocking)

        ppt = getattr(inp, "prefix_page_table", None)
        paged = ppt is not None
        return DeviceInputs(
            q=bf(inp.q), prefix_k=None if paged else bf(inp.prefix_k),
            prefix_v=None if paged else bf(inp.prefix_v),
            prefix_cu=i32(inp.prefix_cu), branch_cu=i32(inp.branch_cu),
            branch_prefix_len=i32(inp.branch_prefix_len), k_cache=bf(inp.k_cache),
            v_cache=bf(inp.v_cache), page_table=i32(inp.page_table),
            branch_len=i32(inp.branch_len), n_docs=inp.n_docs, B=inp.B, m=inp.m, H_q=inp.H_q,
            H_kv=inp.H_kv, D=inp.D, num_pages=inp.num_pages, max_pages=inp.max_pages,
            prefix_tokens=inp.prefix_tokens, max_prefix_len=inp.max_prefix_len,
            scale=float(inp.scale), prefix_page_table=i32(ppt),
            max_prefix_pages=0 if ppt is None else int(ppt.shape[1]))


def make_args(d: DeviceInputs, out=None, lse=None, workspace=None,
              workspace_bytes: int = 0) -> hpd_branch_attn_args:
    a = hpd_branch_attn_args()
    a.q, a.prefix_k, a.prefix_v = _ptr(d.q), _ptr(d.prefix_k), _ptr(d.prefix_v)
    a.prefix_cu, a.branch_cu = _ptr(d.prefix_cu), _ptr(d.branch_cu)
    a.branch_prefix_len = _ptr(d.branch_prefix_len)
    a.k_cache, a.v_cache = _ptr(d.k_cache), _ptr(d.v_cache)
    a.page_table, a.branch_len = _ptr(d.page_table), _ptr(d.branch_len)
    a.n_docs, a.B, a.m, a.H_q, a.H_kv, a.D = d.n_docs, d.B, d.m, d.H_q, d.H_kv, d.D
    a.num_pages, a.max_pages_per_branch = d.num_pages, d.max_pages
    a.prefix_tokens, a.max_prefix_len = d.prefix_tokens, d.max_prefix_len
    a.scale = d.scale
    a.prefix_page_table = _ptr(d.prefix_page_table)
    a.max_prefix_pages = d.max_prefix_pages
    a.out, a.lse = _ptr(out), _ptr(lse)
    a.workspace = _ptr(workspace)
    a.workspace_bytes = int(workspace_bytes)
    return a


class BranchAttn:
    """Owns the output and workspace tensors for repeated calls on one
    workload shape; ``__call__`` enqueues one step on ``stream``."""

    def __init__(self, d: DeviceInputs, stream=None):
        import torch
        self.d = d
        dev = d.q.device
        self.out = torch.empty((d.B * d.m, d.H_q, d.D), dtype=torch.bfloat16, device=dev)
        self.lse = torch.empty((d.B * d.m, d.H_q), dtype=torch.float32, device=dev)
        nbytes = hpd_branch_attn_workspace_size(make_args(d))
        if nbytes == 0:
            raise HpdError("hpd_branch_attn_workspace_size", 1, "invalid shape")
        self.workspace = torch.empty(nbytes, dtype=torch.uint8, device=dev)
        self.args = make_args(d, self.out, self.lse, self.workspace, nbytes)
        hpd_workspace_init(_ptr(self.workspace), nbytes, _stream_handle(stream))

    def rebind(self, d: DeviceInputs):
        """Point the call at another set of inputs of the same shape."""
        self.d = d
        self.args = make_args(d, self.out, self.lse, self.workspace, self.workspace.numel())

    def __call__(self, stream=None, events=None):
        """Enqueue one step; ``events`` (torch.cuda.Event list, launches + 1
        long, already recorded once so their handles exist) marks each kernel."""
        if events is None:
            hpd_branch_attn(self.args, _stream_handle(stream))
        else:
            hpd_branch_attn_marked(self.args, _stream_handle(stream),
                                   [int(e.cuda_event) for e in events])
        return self.out, self.lse

    def step(self, logits, drafts, out_tokens, accepted_len, stream=None):
        """Enqueue one decode step: this attention call and the acceptance of
        ``logits`` (bf16 [B, m, V]) against ``drafts`` (int32 [B, m]) into
        ``out_tokens`` (int32 [B, m]) and ``accepted_len`` (int32 [B])."""
        hpd_decode_step(self.args, _ptr(logits), _ptr(drafts), int(logits.shape[-1]),
                        _ptr(out_tokens), _ptr(accepted_len), _stream_handle(stream))
        return self.out, self.lse

    def errors(self, stream=None) -> int:
        return hpd_read_errors(_ptr(self.workspace), _stream_handle(stream))


def branch_attn(d: DeviceInputs, stream=None):
    """One branch-decode attention step; returns (out bf16, lse fp32)."""
    op = BranchAttn(d, stream)
    return op(stream)


def pmtp_accept(logits, drafts, stream=None):
    """Greedy acceptance on device tensors: logits bf16 [B, m, V], drafts
    int32 [B, m]; returns (out_tokens int32 [B, m], accepted_len int32 [B])."""
    import torch
    B, m, V = logits.shape
    out_tokens = torch.empty((B, m), dtype=torch.int32, device=logits.device)
    acc = torch.empty((B,), dtype=torch.int32, device=logits.device)
    hpd_pmtp_accept(_ptr(logits), _ptr(drafts), B, m, V, _ptr(out_tokens), _ptr(acc),
                    _stream_handle(stream))
    return out_tokens, acc


class PagedKV:
    """Device state of the paged private KV (tensors owned here): the caches,
    the page table, the branch lengths and the free-page stack, plus a
    256-byte workspace for the error word.  append() / rollback() call the
    C ABI on it."""

    def __init__(self, k_cache, v_cache, page_table, branch_len, free_pages, free_top, m):
        import torch
        self.k_cache, self.v_cache = k_cache, v_cache
        self.page_table, self.branch_len = page_table, branch_len
        self.free_pages, self.free_top = free_pages, free_top
        self.m = m
        self.workspace = torch.zeros(256, dtype=torch.uint8, device=k_cache.device)
        B, max_pages = page_table.shape
        num_pages, _, H_kv, D = k_cache.shape
        self.args = hpd_kv_args(None, None, _ptr(k_cache), _ptr(v_cache), _ptr(page_table),
                                _ptr(branch_len), _ptr(free_pages), _ptr(free_top),
                                _ptr(self.workspace), B, m, H_kv, D, num_pages, max_pages)

    def append(self, k_new, v_new, stream=None):
        self.args.k_new, self.args.v_new = _ptr(k_new), _ptr(v_new)
        hpd_kv_append(self.args, _stream_handle(stream))

    def rollback(self, accepted_len, stream=None):
        hpd_kv_rollback(self.args, _ptr(accepted_len), _stream_handle(stream))

    def errors(self, stream=None) -> int:
        return hpd_read_errors(_ptr(self.workspace), _stream_handle(stream))


def fork_children(out_tokens, accepted_len, is_layout, layout_pos, fork_token, branch_cu,
                  branch_prefix_len, branch_len, page_table, cap, stream=None):
    """Device tensors in (int32); returns a dict of new device tensors
    (branch_cu, branch_prefix_len, branch_len, page_table, parent, new_B,
    workspace) with capacity `cap` branches."""
    import torch
    dev = out_tokens.device
    B, m = out_tokens.shape
    n_docs = branch_cu.shape[0] - 1
    max_pages = page_table.shape[1]
    new = dict(branch_cu=torch.empty(n_docs + 1, dtype=torch.int32, device=dev),
               branch_prefix_len=torch.empty(cap, dtype=torch.int32, device=dev),
               branch_len=torch.empty(cap, dtype=torch.int32, device=dev),
               page_table=torch.empty((cap, max_pages), dtype=torch.int32, device=dev),
               parent=torch.empty(cap, dtype=torch.int32, device=dev),
               new_B=torch.empty(1, dtype=torch.int32, device=dev))
    ws_bytes = max(256, 4 * (65 + n_docs))
    ws_bytes = (ws_bytes + 255) // 256 * 256
    new["workspace"] = torch.zeros(ws_bytes, dtype=torch.uint8, device=dev)
    args = hpd_fork_args(_ptr(out_tokens), _ptr(accepted_len), _ptr(is_layout), _ptr(layout_pos),
                         _ptr(branch_cu), _ptr(branch_prefix_len), _ptr(branch_len),
                         _ptr(page_table), _ptr(new["branch_cu"]), _ptr(new["branch_prefix_len"]),
                         _ptr(new["branch_len"]), _ptr(new["page_table"]), _ptr(new["parent"]),
                         _ptr(new["new_B"]), _ptr(new["workspace"]), ws_bytes, fork_token, B, m,
                         n_docs, max_pages, cap)
    _check("hpd_fork_children", load().hpd_fork_children(ctypes.byref(args), _stream_handle(stream)))
    return new
