#!/usr/bin/env python3
"""Benchmark of the branch-decode step of Hierarchical Parallel Decoding.

One step = one pass of the whole hot path over one batch of synthetic input:
hpd_branch_attn (one persistent tcgen05 kernel over every branch's shared
prefix and paged private suffix, preceded by a unit-ordering pass when there
are at least two units per SM and followed by the LSE merge of key splits
when the keys are split) followed by hpd_pmtp_accept (greedy verification of
the P-MTP drafts against bf16 logits over a 32,000-token vocabulary).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload c2]
                    [--impl ours|reference]

Prints ONE JSON line on rank 0.  The metric is query tokens (branches x m)
per second; ``roofline`` reports the dominant kernel against the measured
peaks in MEASURED_PEAKS.json; ``cpu_baseline`` times the fp64 oracle on the
host cores.  ``--impl reference`` times the oracle itself as the bench arm.

Timing: W warm-up steps, then exactly K steps replayed from CUDA graphs,
bracketed by a barrier and a device synchronize, with the input replicas
rotated so that their footprint exceeds 3x the L2 cache.  Per-kernel times
come from timing markers recorded inside the graphs of the timed region.
Under torchrun each rank processes its own pages (pages are independent; no
collective on the data path) and the slowest rank's time is used.
"""
from __future__ import annotations

import argparse
import csv
import glob
import hashlib
import io
import json
import math
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2607_18839_gb300 import workloads as W  # noqa: E402

METRIC = "branch-decode query-tokens/s"
NOMINAL_HBM_GBS = 7900.0      # GB300 HBM3e, nominal
NOMINAL_BF16_TFLOPS = 2250.0  # GB300 dense bf16 tensor, nominal
UNIT = "query-tokens/s"
VOCAB = 32000
DRAFT_MATCH = 0.7
ACCEPT = "pmtp_accept"


# ------------------------------------------------------------------ helpers --

def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return dict(hbm=float(p["hbm_gbs"]), tc_burst=float(p["bf16_tflops"]),
                    tc_sustained=float(p.get("bf16_tflops_sustained", p["bf16_tflops"])),
                    source="measured")
    return dict(hbm=6800.0, tc_burst=1900.0, tc_sustained=1700.0, source="fallback")


def algorithmic_work(inp, V=VOCAB):
    """Algorithmic bytes / FLOPs of one step, per kernel (the unit each
    kernel must move or compute no matter how it is written)."""
    m, Hq, Hkv, D = inp.m, inp.H_q, inp.H_kv, inp.D
    P = np.diff(inp.prefix_cu).astype(np.float64)
    Bd = np.diff(inp.branch_cu).astype(np.float64)
    L = inp.branch_len.astype(np.float64)
    rows = inp.B * m
    q_bytes = rows * Hq * D * 2
    prefix_kv = P.sum() * Hkv * D * 2 * 2
    private_kv = L.sum() * Hkv * D * 2 * 2
    pages_used = np.ceil(L / W.PAGE).sum()
    tables = pages_used * 4 + inp.B * 4 + 2 * (inp.n_docs + 1) * 4
    out_bytes = rows * Hq * D * 2 + rows * Hq * 4
    prefix_flops = 4.0 * (Bd * m * Hq * P).sum() * D
    vis = np.zeros(inp.B)
    for i in range(m):
        vis += np.maximum(0.0, L - m + i + 1)
    suffix_flops = 4.0 * Hq * D * vis.sum()
    accept_bytes = rows * V * 2 + rows * 4 * 2 + inp.B * 4
    per = {
        # tcgen05 path: one kernel for prefix + suffix (+ merge of key splits)
        "branch_attn_tc": dict(bytes=prefix_kv + private_kv + q_bytes + tables + out_bytes,
                               flops=prefix_flops + suffix_flops),
        "merge_splits": dict(bytes=out_bytes, flops=0.0),
        # longest-first order of the work units: the lengths and offsets it reads
        "unit_order": dict(bytes=inp.B * 8 + (inp.n_docs + 1) * 8, flops=0.0),
        # warp-MMA path (G not dividing 128)
        "prefix_stage": dict(bytes=prefix_kv + q_bytes, flops=prefix_flops),
        "suffix_merge": dict(bytes=private_kv + q_bytes + tables + out_bytes, flops=suffix_flops),
        ACCEPT: dict(bytes=accept_bytes, flops=0.0),
    }
    step_bytes = q_bytes + prefix_kv + private_kv + tables + out_bytes + accept_bytes
    return per, dict(bytes=step_bytes, flops=prefix_flops + suffix_flops)


# Sources each kernel is compiled from (its .cu, the headers it includes and
# the host planner that shapes its launch): its recorded DRAM traffic stays
# valid while these are unchanged.
KERNEL_SOURCES = {
    "branch_attn_tc": ["branch_attn_tc.cu", "tc_common.cuh", "sm100.cuh", "common.cuh", "hpd_api.cu"],
    "unit_order": ["unit_order.cu", "common.cuh", "hpd_api.cu"],
    "merge_splits": ["merge.cu", "common.cuh", "hpd_api.cu"],
    "pmtp_accept": ["accept.cu", "common.cuh"],
}


def kernel_source_hash(kernel):
    """Hash of the kernel's sources with comments and blank space removed
    (a documentation edit does not change the kernel)."""
    import re
    h = hashlib.sha256()
    for name in KERNEL_SOURCES.get(kernel, []) + ["../../include/hpd.h"]:
        with open(os.path.join(ROOT, "paper_2607_18839_gb300", "csrc", name)) as f:
            text = f.read()
        text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
        text = re.sub(r"//[^\n]*", " ", text)
        h.update(os.path.basename(name).encode())
        h.update(" ".join(text.split()).encode())
    return h.hexdigest()[:16]


def ncu_traffic(workload, kernel):
    """DRAM bytes per launch of `kernel` from the committed ncu summary, or
    None when there is none or the kernel's sources changed since it was
    taken."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        t = json.load(f)
    e = t.get("workloads", {}).get(workload, {}).get(kernel)
    if e is None or e.get("source_hash") != kernel_source_hash(kernel):
        return None
    return float(e["dram_bytes_per_launch"])


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.gpu_id = gpu_id
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", self.gpu_id, f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.15)

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.1)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        rows = [r for r in csv.reader(io.StringIO(out)) if len(r) >= 9]
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].strip().replace(".", "").isdigit()]
        smax = [float(r[2]) for r in rows if r[2].strip().replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[k] for r in rows for k in range(4)
                          if r[5 + k].strip().lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "reasons": reasons, "samples": len(rows)}


def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def rank_seeds(cid: int, rank: int):
    """Seeds of a rank's workload (tensors, logits).  Every rank runs its own
    independent pages (pages never share keys), so ranks draw distinct data."""
    return 1000 + cid + 100 * rank, 2000 + cid + 100 * rank


def max_over_ranks(ms: float, world: int, device) -> float:
    """The slowest rank's time: all-reduce MAX over the process group."""
    if world <= 1:
        return ms
    import torch
    import torch.distributed as dist
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_value(world: int, qtok_per_rank: int, ms_per_step: float) -> float:
    """Query tokens all ranks processed per second (weak scaling: each rank
    processes qtok_per_rank per step, ms_per_step is the max over ranks)."""
    return world * qtok_per_rank / (ms_per_step * 1e-3)


# ------------------------------------------------------------- CPU oracle --

def oracle_sample_run(inp, logits, drafts, budget_s: float, rng_seed: int = 0):
    """Time the fp64 oracle (attention + acceptance) on a bounded sample of
    the workload: a random subset of branches, all their queries and heads,
    repeated until ``budget_s`` seconds.  Returns (query tokens/s, threads,
    sample description)."""
    import oracle
    per, _ = algorithmic_work(inp)
    est_flops = 2.0 * (per["branch_attn_tc"]["flops"]) / inp.B
    threads = oracle.max_threads()
    per_branch_s = est_flops / (0.5e9 * threads)  # ~0.5 GFLOP/s per thread, fp64 scalar loops
    n = int(max(1, min(inp.B, budget_s / 3.0 / max(per_branch_s, 1e-9))))
    rng = np.random.default_rng(rng_seed)
    sel = np.sort(rng.choice(inp.B, size=n, replace=False)).astype(np.int32)
    rows = (sel[:, None] * inp.m + np.arange(inp.m)).reshape(-1)
    lg = logits[sel]
    dr = drafts[sel]
    reps, t0 = 0, time.perf_counter()
    while True:
        oracle.branch_attn(inp, branch_sel=sel)
        oracle.pmtp_accept(lg, dr)
        reps += 1
        el = time.perf_counter() - t0
        if el >= budget_s or reps >= 1000:
            break
    value = reps * len(rows) / el
    sample = (f"{n} of {inp.B} branches ({len(rows)} query tokens, all heads, full prefix + "
              f"suffix, + acceptance of their {len(rows)} logits rows) x {reps} reps in {el:.1f} s")
    return value, threads, sample


# --------------------------------------------------------------- our path --

def run_ours(args, world, rank, local):
    import torch
    import torch.distributed as dist
    from paper_2607_18839_gb300 import build as hpd_build
    from paper_2607_18839_gb300 import hpd as H

    if not torch.cuda.is_available():
        raise SystemExit("bench.py: no CUDA device (the CUDA path has no CPU fallback)")
    if world > 1:
        dist.init_process_group("nccl", init_method="env://")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    hpd_build.build()
    H.load()

    cid = int(args.workload.lstrip("c"))
    seed_t, seed_l = rank_seeds(cid, rank)
    inp = W.make_config(args.workload, seed=seed_t)
    logits_np = W.make_logits(inp.B, inp.m, VOCAB, seed=seed_l)
    stream = torch.cuda.Stream(device=dev)
    sh = int(stream.cuda_stream)

    # ---- replicas: footprint > 3x L2 so timed steps read from HBM
    base = H.DeviceInputs.from_host(inp, device=dev)
    logits0 = torch.from_numpy(logits_np.view(np.int16)).to(dev).view(torch.bfloat16)
    tensors = [base.q, base.prefix_k, base.prefix_v, base.k_cache, base.v_cache, base.page_table,
               base.branch_len, base.prefix_cu, base.branch_cu, logits0]
    rep_bytes = sum(t.numel() * t.element_size() for t in tensors)
    l2 = int(getattr(torch.cuda.get_device_properties(dev), "L2_cache_size", 128 << 20))
    free, _ = torch.cuda.mem_get_info(dev)
    R = max(2, math.ceil(3 * l2 / rep_bytes))
    R = int(min(R, 256, max(2, (free * 0.5) // rep_bytes)))

    def clone_inputs(d):
        return H.DeviceInputs(**{k: (v.clone() if isinstance(v, torch.Tensor) else v)
                                 for k, v in d.__dict__.items()})

    # (the library keeps raw device pointers: these lists keep the tensors alive)
    reps = [base] + [clone_inputs(base) for _ in range(R - 1)]
    logits = [logits0] + [logits0.clone() for _ in range(R - 1)]
    op = H.BranchAttn(base, stream=stream)
    argsets = [H.make_args(d, op.out, op.lse, op.workspace, op.workspace.numel()) for d in reps]
    n_launch = H.hpd_branch_attn_launches(argsets[0])
    out_tokens = torch.empty((inp.B, inp.m), dtype=torch.int32, device=dev)
    acc = torch.empty((inp.B,), dtype=torch.int32, device=dev)

    # drafts: the row argmax (from this library's first acceptance call) kept
    # with probability 0.7 per position, else a uniform random token
    zeros = torch.zeros((inp.B, inp.m), dtype=torch.int32, device=dev)
    with torch.cuda.stream(stream):
        H.hpd_pmtp_accept(logits0.data_ptr(), zeros.data_ptr(), inp.B, inp.m, VOCAB,
                          out_tokens.data_ptr(), acc.data_ptr(), sh)
    stream.synchronize()
    drafts_np = W.mix_drafts(out_tokens.cpu().numpy(), VOCAB, DRAFT_MATCH, seed=3000 + rank)
    drafts = torch.from_numpy(drafts_np).to(dev)

    def attn(r, ev=None):
        if ev is None:
            H.hpd_branch_attn(argsets[r], sh)
        else:
            H.hpd_branch_attn_marked(argsets[r], sh, ev)

    def accept(r):
        H.hpd_pmtp_accept(logits[r].data_ptr(), drafts.data_ptr(), inp.B, inp.m, VOCAB,
                          out_tokens.data_ptr(), acc.data_ptr(), sh)

    def step(r, ev=None):
        attn(r, ev)
        accept(r)

    # ---- warm-up (eager), also sets the kernels' function attributes
    with torch.cuda.stream(stream):
        for i in range(max(args.warmup, 3)):
            step(i % R)
    stream.synchronize()
    err = op.errors(stream)
    if err:
        raise SystemExit(f"bench.py: device error flags {err:#x}")

    # ---- CUDA graphs of S steps (inputs rotated over the R replicas)
    K = args.steps
    S = max(1, min(K, args.graph_steps))

    def capture(nsteps, offset, body):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for i in range(nsteps):
                body((offset + i) % R, i)
        return g

    g_main = capture(S, 0, lambda r, i: step(r))
    g_rem = capture(K % S, S, lambda r, i: step(r)) if K % S else None
    n_main = K // S

    wall_ms = [0.0]  # host wall clock of the last timed region (cross-check)

    def timed(gm, gr, nm, sync_ranks=True):
        if world > 1 and sync_ranks:
            dist.barrier()
        torch.cuda.synchronize(dev)
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        w0 = time.perf_counter()
        # replay() launches on the current stream: make it the timing stream
        with torch.cuda.stream(stream):
            t0.record(stream)
            for _ in range(nm):
                gm.replay()
            if gr is not None:
                gr.replay()
            t1.record(stream)
        torch.cuda.synchronize(dev)
        wall_ms[0] = (time.perf_counter() - w0) * 1e3
        ms = t0.elapsed_time(t1)
        if world > 1 and sync_ranks:
            ms = max_over_ranks(ms, world, dev)
            dist.barrier()
        return ms

    gpu_id = str(torch.cuda.get_device_properties(dev).uuid)
    gpu_id = gpu_id if gpu_id.startswith("GPU-") else f"GPU-{gpu_id}"
    clocks = ClockSampler(gpu_id)
    clocks.start()
    total_ms = timed(g_main, g_rem, n_main)
    total_wall_ms = wall_ms[0]
    clk = clocks.stop()

    # ---- per-kernel durations, measured right after the timed region on the
    # same stream: the attention call and the acceptance kernel each replayed
    # back to back from their own graphs (events around the replays), and the
    # attention call's kernels apportioned by timing markers recorded inside a
    # graph of marked calls.
    n_rep = max(1, (2 * K) // S)
    g_attn = capture(S, 0, lambda r, i: attn(r))
    g_acc = capture(S, 0, lambda r, i: accept(r))
    attn_ms = timed(g_attn, None, n_rep, sync_ranks=False) / (n_rep * S)
    acc_ms = timed(g_acc, None, n_rep, sync_ranks=False) / (n_rep * S)
    attn_names = [H.hpd_branch_attn_kernel_name(argsets[0], k) for k in range(n_launch)]
    events = [[torch.cuda.Event(enable_timing=True) for _ in range(n_launch + 1)] for _ in range(S)]
    with torch.cuda.stream(stream):
        for row in events:
            for e in row:
                e.record(stream)  # creates the handle
    stream.synchronize()
    handles = [[int(e.cuda_event) for e in row] for row in events]
    g_mark = capture(S, 0, lambda r, i: attn(r, handles[i]))
    with torch.cuda.stream(stream):
        g_mark.replay()
    torch.cuda.synchronize(dev)
    span = [statistics.mean(ev[k].elapsed_time(ev[k + 1]) for ev in events) for k in range(n_launch)]
    kernel_ms = {name: attn_ms * span[k] / sum(span) for k, name in enumerate(attn_names)}
    kernel_ms[ACCEPT] = acc_ms

    # ---- paged-KV append / rollback around a step (reported beside the step,
    # not part of its metric): append the step's m rows of every branch, then
    # roll all of them back (accepted_len = -1), which restores the pool
    used = np.ceil(inp.branch_len / W.PAGE).astype(np.int64)
    kv_max_pages = int(np.max(np.ceil((inp.branch_len + inp.m) / W.PAGE)))
    kv_pages = int(used.sum() + inp.B * (inp.m // W.PAGE + 2))
    pool = W.make_kv_pool(inp.branch_len, inp.m, inp.H_kv, inp.D, kv_pages, kv_max_pages,
                          seed=4000 + cid)
    kv_new = W.make_kv_rows(inp.B, inp.m, inp.H_kv, inp.D, seed=5000 + cid)
    tdev = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    kv = H.PagedKV(tdev(pool["k_cache"].view(np.int16)), tdev(pool["v_cache"].view(np.int16)),
                   tdev(pool["page_table"]), tdev(pool["branch_len"]), tdev(pool["free"]),
                   torch.tensor([pool["top"]], dtype=torch.int32, device=dev), inp.m)
    k_new, v_new = (tdev(a.view(np.int16)) for a in kv_new)
    reject_all = torch.full((inp.B,), -1, dtype=torch.int32, device=dev)

    def kv_pair(r, i):
        kv.append(k_new, v_new, stream)
        kv.rollback(reject_all, stream)

    with torch.cuda.stream(stream):
        kv_pair(0, 0)
    g_kv = capture(S, 0, kv_pair)
    kv_ms = timed(g_kv, None, n_rep, sync_ranks=False) / (n_rep * S)
    if kv.errors(stream):
        raise SystemExit(f"bench.py: KV append / rollback error flags {kv.errors(stream):#x}")
    kv_bytes = 2 * 2 * inp.B * inp.m * inp.H_kv * inp.D * 2  # K and V rows read + written
    kv_line = {"us_per_pair": kv_ms * 1e3, "launches_per_pair": 3, "bytes": kv_bytes,
               "achieved_gbs": kv_bytes / (kv_ms * 1e-3) / 1e9,
               "note": "hpd_kv_append (m rows per branch) + hpd_kv_rollback (all rolled back) "
                       "on a pool of the workload's lengths; not part of the step metric"}

    # ---- fork detection / child branches after the acceptance (reported beside
    # the step): the step's argmax tokens with 2% fork tokens, each page's
    # first branch its layout branch
    rng_f = np.random.default_rng(6000 + cid)
    fork_tok = np.where(rng_f.random((inp.B, inp.m)) < 0.02, VOCAB - 1,
                        rng_f.integers(0, VOCAB - 1, size=(inp.B, inp.m))).astype(np.int32)
    is_layout = np.zeros(inp.B, np.int32)
    is_layout[inp.branch_cu[:-1][np.diff(inp.branch_cu) > 0]] = 1
    f_in = [tdev(a) for a in (fork_tok, acc.cpu().numpy(), is_layout,
                               inp.branch_prefix_len if inp.branch_prefix_len is not None
                               else np.zeros(inp.B, np.int32), inp.branch_cu, inp.branch_len,
                               inp.page_table)]
    f_cap = inp.B * (inp.m + 1)
    f_state = {}

    def fork_call(r, i):
        f_state["out"] = H.fork_children(f_in[0], f_in[1], f_in[2], f_in[3], VOCAB - 1, f_in[4],
                                         None, f_in[5], f_in[6], f_cap, stream)

    with torch.cuda.stream(stream):
        fork_call(0, 0)
    torch.cuda.synchronize(dev)
    g_fork = capture(S, 0, fork_call)
    fork_ms = timed(g_fork, None, n_rep, sync_ranks=False) / (n_rep * S)
    fork_line = {"us_per_call": fork_ms * 1e3,
                 "children": int(f_state["out"]["new_B"].item()) - inp.B,
                 "note": "hpd_fork_children over the step's branches (two launches); not part of "
                         "the step metric"}

    # ---- the attention call on other layouts of the prefix and on the
    # layout-branch workload (reported beside the step; one input replica)
    def attn_call_us(inp_x):
        op_x = H.BranchAttn(H.DeviceInputs.from_host(inp_x), stream)
        with torch.cuda.stream(stream):
            for _ in range(3):
                op_x(stream)
        torch.cuda.synchronize(dev)
        g_x = capture(S, 0, lambda r, i: op_x(stream))
        ms = timed(g_x, None, n_rep, sync_ranks=False) / (n_rep * S)
        if op_x.errors(stream):
            raise SystemExit(f"bench.py: error flags {op_x.errors(stream):#x} on {inp_x.name}")
        return ms * 1e3, H.hpd_branch_attn_launches(op_x.args)

    runs_us, _ = attn_call_us(W.page_the_prefix(inp, seed=7000 + cid, runs=True))
    scat_us, _ = attn_call_us(W.page_the_prefix(inp, seed=7000 + cid, runs=False))
    paged_line = {"us_per_call_consecutive_pages": runs_us, "us_per_call_scattered_pages": scat_us,
                  "contiguous_us_per_call": attn_ms * 1e3,
                  "note": "the same attention call with every page's prefix in the 16-token KV "
                          "pool through a prefix page table: in consecutive pool pages (one "
                          "prefill allocation) or scattered; one L2-warm input replica"}
    lay = W.make_layout_config()
    lay_us, lay_launch = attn_call_us(lay)
    layout_line = {"workload": "8 pages, vision U[1024,3072], layout tokens U[64,512], each "
                               "page's layout branch + U[4,24] content branches forked after "
                               "a layout token (lognormal histories), m=4, Hq16/Hkv2, D128, "
                               "paged prefix shared with the layout branch",
                   "us_per_call": lay_us, "launches": lay_launch,
                   "query_tokens_per_s": lay.B * lay.m / (lay_us * 1e-6),
                   "note": "attention call only, one L2-warm input replica"}

    # ---- end to end: pinned host inputs in, results out, every step.  Each
    # step copies its inputs H2D in one packed copy (q, page table, lengths,
    # offsets, logits, drafts), runs the attention and the acceptance through
    # the C ABI, and copies its results D2H in one packed copy (out, lse,
    # tokens, accepted lengths).  Two slots and three streams (H2D, compute,
    # D2H) let a step's copies overlap the neighbouring steps' kernels; the
    # resident prefix and paged KV rotate over the replicas as above.
    def packed(sizes):
        offs, o = [], 0
        for n in sizes:
            offs.append(o)
            o += (n + 255) // 256 * 256
        return offs, o

    in_arrays = [np.ascontiguousarray(a) for a in (inp.q, inp.page_table.astype(np.int32),
                                                    inp.branch_len.astype(np.int32),
                                                    inp.prefix_cu.astype(np.int32),
                                                    inp.branch_cu.astype(np.int32), logits_np,
                                                    drafts_np.astype(np.int32))]
    in_sizes = [a.nbytes for a in in_arrays]
    in_offs, in_total = packed(in_sizes)
    host_in = torch.zeros(in_total, dtype=torch.uint8).pin_memory()
    for arr, o in zip(in_arrays, in_offs):
        host_in[o:o + arr.nbytes].copy_(torch.from_numpy(arr.reshape(-1).view(np.uint8)))
    rows = inp.B * inp.m
    out_sizes = [rows * inp.H_q * inp.D * 2, rows * inp.H_q * 4, rows * 4, inp.B * 4]
    out_offs, out_total = packed(out_sizes)
    host_out = torch.empty(out_total, dtype=torch.uint8).pin_memory()

    def view(buf, off, n, dtype, shape):
        return buf[off:off + n].view(dtype).view(shape)

    slots = []
    for _ in range(2):
        din = torch.empty(in_total, dtype=torch.uint8, device=dev)
        dout = torch.empty(out_total, dtype=torch.uint8, device=dev)
        i32 = torch.int32
        slots.append(dict(
            din=din, dout=dout,
            q=view(din, in_offs[0], in_sizes[0], torch.bfloat16, (rows, inp.H_q, inp.D)),
            pt=view(din, in_offs[1], in_sizes[1], i32, inp.page_table.shape),
            bl=view(din, in_offs[2], in_sizes[2], i32, (inp.B,)),
            pcu=view(din, in_offs[3], in_sizes[3], i32, (inp.n_docs + 1,)),
            bcu=view(din, in_offs[4], in_sizes[4], i32, (inp.n_docs + 1,)),
            lg=view(din, in_offs[5], in_sizes[5], torch.bfloat16, (inp.B, inp.m, VOCAB)),
            dr=view(din, in_offs[6], in_sizes[6], i32, (inp.B, inp.m)),
            out=view(dout, out_offs[0], out_sizes[0], torch.bfloat16, (rows, inp.H_q, inp.D)),
            lse=view(dout, out_offs[1], out_sizes[1], torch.float32, (rows, inp.H_q)),
            tok=view(dout, out_offs[2], out_sizes[2], i32, (inp.B, inp.m)),
            acc=view(dout, out_offs[3], out_sizes[3], i32, (inp.B,))))
    e2e_args = {}

    def slot_args(s_i, r):
        if (s_i, r) not in e2e_args:
            sl, rep = slots[s_i], reps[r]
            d = H.DeviceInputs(**{**rep.__dict__, "q": sl["q"], "page_table": sl["pt"],
                                  "branch_len": sl["bl"], "prefix_cu": sl["pcu"],
                                  "branch_cu": sl["bcu"]})
            e2e_args[(s_i, r)] = (d, H.make_args(d, sl["out"], sl["lse"], op.workspace,
                                                 op.workspace.numel()))
        return e2e_args[(s_i, r)][1]

    h2d_s = torch.cuda.Stream(device=dev)
    d2h_s = torch.cuda.Stream(device=dev)

    def e2e_capture(nsteps, offset):
        g = torch.cuda.CUDAGraph()
        events = []  # keep the events alive with the graph
        with torch.cuda.graph(g, stream=stream):
            h2d_s.wait_stream(stream)
            d2h_s.wait_stream(stream)
            comp, out_done = {}, {}
            for i in range(nsteps):
                s_i, r = i % 2, (offset + i) % R
                sl = slots[s_i]
                ev_in = torch.cuda.Event()
                with torch.cuda.stream(h2d_s):
                    if i >= 2:
                        h2d_s.wait_event(comp[i - 2])   # the slot's inputs were consumed
                    sl["din"].copy_(host_in, non_blocking=True)
                    ev_in.record(h2d_s)
                stream.wait_event(ev_in)
                if i >= 2:
                    stream.wait_event(out_done[i - 2])  # the slot's results were read out
                H.hpd_branch_attn(slot_args(s_i, r), sh)
                H.hpd_pmtp_accept(sl["lg"].data_ptr(), sl["dr"].data_ptr(), inp.B, inp.m, VOCAB,
                                  sl["tok"].data_ptr(), sl["acc"].data_ptr(), sh)
                comp[i] = torch.cuda.Event()
                comp[i].record(stream)
                with torch.cuda.stream(d2h_s):
                    d2h_s.wait_event(comp[i])
                    host_out.copy_(sl["dout"], non_blocking=True)
                    out_done[i] = torch.cuda.Event()
                    out_done[i].record(d2h_s)
                events += [ev_in, comp[i], out_done[i]]
            stream.wait_stream(h2d_s)
            stream.wait_stream(d2h_s)
        g._hpd_events = events
        return g

    h2d_bytes = sum(in_sizes)
    d2h_bytes = sum(out_sizes)
    ge_main = e2e_capture(S, 0)
    ge_rem = e2e_capture(K % S, S) if K % S else None
    with torch.cuda.stream(stream):
        ge_main.replay()  # untimed first replay
    torch.cuda.synchronize(dev)
    e2e_ms = timed(ge_main, ge_rem, n_main)
    err = op.errors(stream)
    if err:
        raise SystemExit(f"bench.py: device error flags {err:#x}")
    # the results that came back are the library's (the last replayed step's slot)
    last = slots[((K % S) - 1) % 2] if ge_rem is not None else slots[(S - 1) % 2]
    if not torch.equal(host_out, last["dout"].cpu()):
        raise SystemExit("bench.py: end-to-end results differ from the device copy")

    # ---- CPU baseline: the oracle on this host's cores (rank 0, N = 1 only)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        v, thr, sample = oracle_sample_run(inp, logits_np, drafts_np, args.cpu_seconds)
        cpu = {"value": v, "unit": UNIT, "cores": thr, "kind": "oracle", "sample": sample}

    if world > 1:
        dist.destroy_process_group()
    if rank != 0:
        return None

    qtok = inp.B * inp.m
    ms_step = total_ms / K
    value = whole_job_value(world, qtok, ms_step)
    e2e_value = whole_job_value(world, qtok, e2e_ms / K)

    pk = peaks()
    per, step_work = algorithmic_work(inp)
    known = {k: v for k, v in kernel_ms.items() if v is not None}
    dom = max(known, key=known.get)
    dom_ms = known[dom]
    t_bytes = per[dom]["bytes"] / (pk["hbm"] * 1e9)
    t_flops = per[dom]["flops"] / (pk["tc_sustained"] * 1e12)
    if t_flops > t_bytes:
        achieved = per[dom]["flops"] / (dom_ms * 1e-3) / 1e12
        roof = {"bound": "tensor", "achieved": achieved, "peak": pk["tc_sustained"],
                "unit": "TFLOP/s"}
    else:
        achieved = per[dom]["bytes"] / (dom_ms * 1e-3) / 1e9
        roof = {"bound": "hbm", "achieved": achieved, "peak": pk["hbm"], "unit": "GB/s"}
    roof["frac"] = roof["achieved"] / roof["peak"]
    roof["traffic"] = ncu_traffic(args.workload, dom)
    roof["kernel"] = dom
    roof["peak_source"] = pk["source"] + (" sustained bf16" if roof["bound"] == "tensor" else " HBM copy")
    roof["nominal_peak"] = NOMINAL_BF16_TFLOPS if roof["bound"] == "tensor" else NOMINAL_HBM_GBS
    roof["frac_of_nominal"] = roof["achieved"] / roof["nominal_peak"]
    acc_us = kernel_ms[ACCEPT] * 1e3
    accept_line = {"us_per_call": acc_us, "bytes": per[ACCEPT]["bytes"],
                   "achieved_gbs": per[ACCEPT]["bytes"] / (acc_us * 1e-6) / 1e9,
                   "frac_of_measured_hbm": per[ACCEPT]["bytes"] / (acc_us * 1e-6) / 1e9 / pk["hbm"],
                   "note": "greedy acceptance, HBM-bound: logits read once"}
    t_roof = max(step_work["bytes"] / (pk["hbm"] * 1e9), step_work["flops"] / (pk["tc_sustained"] * 1e12))

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K,
        "warmup": max(args.warmup, 3), "ms_per_step": ms_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {
            "workload": f"{args.workload}: {W.CONFIG_DESCRIPTIONS[args.workload]}; acceptance "
                        f"over bf16 logits [{inp.B} x {inp.m} x {VOCAB}]",
            "query_tokens_per_step": qtok,
            "l2": f"{R} rotating input replicas ({R * rep_bytes / 2**20:.0f} MiB > 3x L2 "
                  f"{l2 / 2**20:.0f} MiB)",
            "timing": f"CUDA graphs of {S} steps, events on the launch stream; per-kernel "
                      f"times from back-to-back graphs of each call after the timed region",
            "parallelism": f"dp{world} (independent pages per GPU, no collective)",
        },
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d_bytes,
                "d2h_bytes_per_step": d2h_bytes,
                "note": "every step: q, page table, lengths, offsets, logits and drafts H2D "
                        "from pinned host memory in one packed copy, out, lse, tokens and "
                        "accepted lengths D2H in one packed copy; two slots on H2D / compute "
                        "/ D2H streams overlap a step's copies with the neighbouring steps' "
                        "kernels; prefix KV and paged KV cache resident"},
        "gpu_launches": K * (n_launch + 1),
        "roofline": roof,
        "step_roofline": {"bytes": step_work["bytes"], "flops": step_work["flops"],
                          "t_roofline_us": t_roof * 1e6,
                          "frac": t_roof / (ms_step * 1e-3)},
        "kernel_us": {k: v * 1e3 for k, v in kernel_ms.items()},
        "attn_call_us": attn_ms * 1e3,
        "accept": accept_line,
        "kv_append_rollback": kv_line,
        "fork_children": fork_line,
        "paged_prefix": paged_line,
        "layout_branches": layout_line,
        "host_wall_ms_per_step": total_wall_ms / K,
        "cpu_baseline": cpu,
        "clocks": clk,
    }
    return line


# --------------------------------------------------------- reference arm --

def run_reference(args, world, rank):
    """The fp64 oracle as the bench arm: each step runs it on a bounded
    sample of the workload on this host's cores."""
    if world > 1 and rank != 0:
        return None
    import oracle
    inp = W.make_config(args.workload)
    cid = int(args.workload.lstrip("c"))
    logits = W.make_logits(inp.B, inp.m, VOCAB, seed=2000 + cid)
    tok, _ = oracle.pmtp_accept(logits, np.zeros((inp.B, inp.m), np.int32))
    drafts = W.mix_drafts(tok, VOCAB, DRAFT_MATCH, seed=3000)
    per, _ = algorithmic_work(inp)
    threads = oracle.max_threads()
    est = 2.0 * (per["branch_attn_tc"]["flops"]) / inp.B
    n = int(max(1, min(inp.B, args.ref_step_seconds / max(est / (0.5e9 * threads), 1e-9))))
    rng = np.random.default_rng(0)
    sel = np.sort(rng.choice(inp.B, size=n, replace=False)).astype(np.int32)
    lg, dr = logits[sel], drafts[sel]
    qtok = n * inp.m

    def step():
        oracle.branch_attn(inp, branch_sel=sel)
        oracle.pmtp_accept(lg, dr)

    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    el = time.perf_counter() - t0
    value = args.steps * qtok / el
    sample = f"{n} of {inp.B} branches ({qtok} query tokens, all heads) + their acceptance rows per step"
    return {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": el / args.steps * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": f"{args.workload}: {W.CONFIG_DESCRIPTIONS[args.workload]}; acceptance "
                               f"over bf16 logits [{inp.B} x {inp.m} x {VOCAB}]",
                   "parallelism": "host CPU (OpenMP)"},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--workload", choices=W.CONFIG_NAMES, default="c2")
    ap.add_argument("--graph-steps", type=int, default=200, help="steps captured per CUDA graph")
    ap.add_argument("--cpu-seconds", type=float, default=10.0, help="oracle CPU-baseline budget")
    ap.add_argument("--ref-step-seconds", type=float, default=1.0,
                    help="oracle work per step of --impl reference")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args()
    world, rank, local = dist_env()
    if args.impl == "reference":
        line = run_reference(args, world, rank)
    else:
        line = run_ours(args, world, rank, local)
    if line is not None and rank == 0:
        print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
