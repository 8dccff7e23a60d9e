"""fp64 CPU oracle for the branch-decode step -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import this package.  The CUDA
library never loads it, and it shares no code with the CUDA library.

The arithmetic lives in ``hpd_oracle.c`` (plain loops in double precision);
this module only compiles it with gcc (on first use, or via :func:`build`)
and marshals numpy arrays into it.

Functions
---------
branch_attn(inp, branch_sel=None, n_threads=0) -> (out fp64, lse fp64)
    Masked-softmax attention of every branch over its shared prefix plus its
    own causal private suffix (Sec. 3.3, "Dynamic Branch Forking and Efficient
    Context Isolation"; Sec. 3.4 for the m P-MTP queries).  The prefix is
    contiguous, or paged in the private keys' pool when the workload carries
    a ``prefix_page_table``.
pmtp_accept(logits_bf16, drafts) -> (out_tokens int32, accepted_len int32)
    Greedy verification of the P-MTP drafts (Sec. 3.4; Algorithm 1's
    verification step), lowest index on argmax ties.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "hpd_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile hpd_oracle.c into liboracle.so (gcc, OpenMP); return its path."""
    stale = (not os.path.exists(_LIB)) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC)
    if force or stale:
        tmp = _LIB + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-fopenmp", "-fPIC", "-shared", "-std=c11",
               "-o", tmp, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        I = ctypes.c_int
        lib.oracle_branch_attn.restype = I
        lib.oracle_branch_attn.argtypes = [P] * 10 + [I] * 8 + [ctypes.c_double, P, I, I, P, P,
                                                                 P, I]
        lib.oracle_pmtp_accept.restype = None
        lib.oracle_pmtp_accept.argtypes = [P, P, I, I, I, P, P]
        lib.oracle_max_threads.restype = I
        lib.oracle_max_threads.argtypes = []
        _lib = lib
    return _lib


def max_threads() -> int:
    """Threads the oracle's OpenMP loop uses by default."""
    return _load().oracle_max_threads()


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return None if a is None else np.ascontiguousarray(a, dtype=dtype)


def branch_attn(inp, branch_sel=None, n_threads: int = 0):
    """Run the oracle on a workload object (see ``workloads.BranchDecodeInputs``).

    Returns ``(out, lse)`` as float64 arrays of shape ``[B*m, H_q, D]`` and
    ``[B*m, H_q]``.  With ``branch_sel`` only those branches' rows are
    computed; the other rows are left as NaN.
    """
    lib = _load()
    rows = inp.B * inp.m
    out = np.full((rows, inp.H_q, inp.D), np.nan, dtype=np.float64)
    lse = np.full((rows, inp.H_q), np.nan, dtype=np.float64)
    arrs = dict(
        q=_c(inp.q, np.uint16), pk=_c(inp.prefix_k, np.uint16), pv=_c(inp.prefix_v, np.uint16),
        pcu=_c(inp.prefix_cu, np.int32), bcu=_c(inp.branch_cu, np.int32),
        bpl=_c(inp.branch_prefix_len, np.int32),
        kc=_c(inp.k_cache, np.uint16), vc=_c(inp.v_cache, np.uint16),
        pt=_c(inp.page_table, np.int32), bl=_c(inp.branch_len, np.int32),
        sel=_c(branch_sel, np.int32),
        ppt=_c(getattr(inp, "prefix_page_table", None), np.int32),
    )
    scale = inp.scale if inp.scale else 1.0 / np.sqrt(inp.D)
    n_sel = 0 if branch_sel is None else len(arrs["sel"])
    rc = lib.oracle_branch_attn(
        _ptr(arrs["q"]), _ptr(arrs["pk"]), _ptr(arrs["pv"]), _ptr(arrs["pcu"]), _ptr(arrs["bcu"]),
        _ptr(arrs["bpl"]), _ptr(arrs["kc"]), _ptr(arrs["vc"]), _ptr(arrs["pt"]), _ptr(arrs["bl"]),
        inp.n_docs, inp.B, inp.m, inp.H_q, inp.H_kv, inp.D, inp.num_pages, inp.max_pages,
        float(scale), _ptr(arrs["sel"]), n_sel, int(n_threads), _ptr(out), _ptr(lse),
        _ptr(arrs["ppt"]), 0 if arrs["ppt"] is None else int(arrs["ppt"].shape[1]))
    if rc != 0:
        raise ValueError("oracle_branch_attn: an index falls outside its buffer")
    return out, lse


def pmtp_accept(logits_bf16: np.ndarray, drafts: np.ndarray):
    """Greedy acceptance; ``logits_bf16`` is uint16 bf16 bits ``[B, m, V]``."""
    lib = _load()
    lg = np.ascontiguousarray(logits_bf16, dtype=np.uint16)
    dr = np.ascontiguousarray(drafts, dtype=np.int32)
    B, m, V = lg.shape
    assert dr.shape == (B, m)
    out_tokens = np.zeros((B, m), dtype=np.int32)
    acc = np.zeros((B,), dtype=np.int32)
    lib.oracle_pmtp_accept(_ptr(lg), _ptr(dr), B, m, V, _ptr(out_tokens), _ptr(acc))
    return out_tokens, acc
