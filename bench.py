#!/usr/bin/env python3
"""Benchmark of the branch-decode step of Hierarchical Parallel Decoding.

One step = one pass of the whole hot path over one batch of synthetic input:
hpd_branch_attn (one persistent tcgen05 kernel over every branch's shared
prefix and paged private suffix, preceded by a unit-ordering pass when there
are at least two units per SM and followed by the LSE merge of key splits
when the keys are split) followed by hpd_pmtp_accept (greedy verification of
the P-MTP drafts against bf16 logits over a 32,000-token vocabulary).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload c4]
                    [--also c2,c3,c5] [--replays 5] [--impl ours|reference]

Prints ONE JSON line on rank 0.  The headline workload is c4 (32 pages, 768
branches, m = 8: the largest single-GPU preset by query tokens and bytes);
the other presets follow in ``per_config``.  The metric is query tokens
(branches x m) per second of the whole step, attention then acceptance;
``attention_only`` gives the attention call alone.  ``roofline`` reports the
dominant kernel against the measured peaks in MEASURED_PEAKS.json;
``cpu_baseline`` times the fp64 oracle on the host cores; ``context`` quotes
the paper's own end-to-end figure.  ``--impl reference`` times the oracle
itself as the bench arm.

Timing: W warm-up steps, then one CUDA graph of exactly K steps replayed at
least five times, each replay bracketed by a barrier and a device
synchronize and timed with CUDA events on the launch stream; the median is
reported.  The input replicas rotate so that their footprint exceeds 3x the
L2 cache; ``cold_l2`` adds steps that each follow an explicit L2 eviction.
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
    Bd = np.diff(inp.branch_cu).astype(np.int64)
    L = inp.branch_len.astype(np.float64)
    # prefix keys each branch sees (its fork-position length, else its page's)
    Pb = np.repeat(P, Bd)
    if inp.branch_prefix_len is not None:
        Pb = np.minimum(Pb, inp.branch_prefix_len.astype(np.float64))
    # per page, the prefix keys some branch of it sees (read once)
    P_read = np.array([Pb[inp.branch_cu[d]:inp.branch_cu[d + 1]].max(initial=0.0)
                       for d in range(inp.n_docs)])
    rows = inp.B * m
    q_bytes = rows * Hq * D * 2
    prefix_kv = P_read.sum() * Hkv * D * 2 * 2
    private_kv = L.sum() * Hkv * D * 2 * 2
    pages_used = np.ceil(L / W.PAGE).sum()
    tables = pages_used * 4 + inp.B * 4 + 2 * (inp.n_docs + 1) * 4
    out_bytes = rows * Hq * D * 2 + rows * Hq * 4
    prefix_flops = 4.0 * m * Hq * D * Pb.sum()
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

PAPER_CONTEXT = {
    "value": 4752.1, "unit": "tokens/s",
    "what": "HPD-Parsing end-to-end decode throughput of the whole model (Table 2)",
    "hardware": "NVIDIA A800 80GB GPUs (count unstated), vLLM 0.17.1, batch 512, OmniDocBench v1.6",
    "note": "context only: another metric (generated tokens of the full model) on other hardware",
}


def step_config(name, world):
    """The `config` object of a workload's bench line (the same in both arms)."""
    inp_desc = W.CONFIG_DESCRIPTIONS[name]
    cfg = W.config_shape(name)
    return {
        "workload": f"{name}: {inp_desc}; acceptance over bf16 logits "
                    f"[{cfg['B']} x {cfg['m']} x {VOCAB}]",
        "query_tokens_per_step": cfg["B"] * cfg["m"],
        "step": "hpd_decode_step: hpd_branch_attn (shared prefix + private suffix + merge) and "
                "hpd_pmtp_accept (acceptance inside the step; it reads only the logits and drafts, "
                "so it runs beside the attention when the attention has fewer than two work units "
                "per SM and leaves SMs idle, else after it)",
        "parallelism": f"dp{world} (independent pages per GPU, no collective)",
    }


class Timer:
    """CUDA-event timing of graph replays on one stream."""

    def __init__(self, torch, dev, stream, world, dist):
        self.torch, self.dev, self.stream, self.world, self.dist = torch, dev, stream, world, dist
        self.wall_ms = 0.0

    def replay_ms(self, graphs, sync_ranks=True):
        """Time one replay of `graphs` (in order), bracketed by a barrier and
        a device synchronize; the max over ranks."""
        torch = self.torch
        if self.world > 1 and sync_ranks:
            self.dist.barrier()
        torch.cuda.synchronize(self.dev)
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        w0 = time.perf_counter()
        with torch.cuda.stream(self.stream):  # replay() launches on the current stream
            t0.record(self.stream)
            for g in graphs:
                g.replay()
            t1.record(self.stream)
        torch.cuda.synchronize(self.dev)
        self.wall_ms = (time.perf_counter() - w0) * 1e3
        ms = t0.elapsed_time(t1)
        if self.world > 1 and sync_ranks:
            ms = max_over_ranks(ms, self.world, self.dev)
            self.dist.barrier()
        return ms

    def median_ms(self, graphs, n, sync_ranks=False):
        return statistics.median(self.replay_ms(graphs, sync_ranks) for _ in range(n))


def measure_workload(name, args, world, rank, dev, stream, H, headline):
    """Time one workload's step (and, for the headline, its side lines)."""
    import torch
    import torch.distributed as dist

    cid = int(name.lstrip("c"))
    seed_t, seed_l = rank_seeds(cid, rank)
    inp = W.make_config(name, seed=seed_t)
    logits_np = W.make_logits(inp.B, inp.m, VOCAB, seed=seed_l)
    sh = int(stream.cuda_stream)
    timer = Timer(torch, dev, stream, world, dist)
    K = args.steps
    n_rep = max(5, args.replays)

    # ---- replicas: footprint > 3x L2 so timed steps read from HBM
    base = H.DeviceInputs.from_host(inp, device=dev)
    logits0 = torch.from_numpy(logits_np.view(np.int16)).to(dev).view(torch.bfloat16)
    tensors = [base.q, base.prefix_k, base.prefix_v, base.k_cache, base.v_cache, base.page_table,
               base.branch_len, base.prefix_cu, base.branch_cu, logits0]
    rep_bytes = sum(t.numel() * t.element_size() for t in tensors)
    l2 = int(getattr(torch.cuda.get_device_properties(dev), "L2_cache_size", 128 << 20))
    free, _ = torch.cuda.mem_get_info(dev)
    R = max(2, math.ceil(3 * l2 / rep_bytes))
    R = int(min(R, 256, max(2, (free * 0.4) // rep_bytes)))

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
    argmax_np = out_tokens.cpu().numpy()
    drafts_np = W.mix_drafts(argmax_np, VOCAB, DRAFT_MATCH, seed=3000 + rank)
    drafts = torch.from_numpy(drafts_np).to(dev)

    def attn(r, ev=None):
        if ev is None:
            H.hpd_branch_attn(argsets[r], sh)
        else:
            H.hpd_branch_attn_marked(argsets[r], sh, ev)

    def accept(r):
        H.hpd_pmtp_accept(logits[r].data_ptr(), drafts.data_ptr(), inp.B, inp.m, VOCAB,
                          out_tokens.data_ptr(), acc.data_ptr(), sh)

    # one step: hpd_decode_step (the attention, and the acceptance beside it
    # when the attention leaves SMs idle, else after it)
    def step(r):
        H.hpd_decode_step(argsets[r], logits[r].data_ptr(), drafts.data_ptr(), VOCAB,
                          out_tokens.data_ptr(), acc.data_ptr(), sh)

    # ---- warm-up (eager), also sets the kernels' function attributes
    with torch.cuda.stream(stream):
        for i in range(max(args.warmup, 3)):
            step(i % R)
    stream.synchronize()
    err = op.errors(stream)
    if err:
        raise SystemExit(f"bench.py: device error flags {err:#x} on {name}")

    def capture(nsteps, offset, body):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for i in range(nsteps):
                body((offset + i) % R, i)
        return g

    # ---- the timed region: one CUDA graph of exactly K steps (inputs
    # rotated over the R replicas), replayed n_rep times; each replay is
    # bracketed by a barrier and a device synchronize, and the median is kept
    g_step = capture(K, 0, lambda r, i: step(r))
    with torch.cuda.stream(stream):
        g_step.replay()  # untimed first replay
    clocks = None
    if headline:
        gpu_id = str(torch.cuda.get_device_properties(dev).uuid)
        gpu_id = gpu_id if gpu_id.startswith("GPU-") else f"GPU-{gpu_id}"
        clocks = ClockSampler(gpu_id)
        clocks.start()
    step_runs = [timer.replay_ms([g_step], sync_ranks=True) for _ in range(n_rep)]
    wall_ms = timer.wall_ms
    clk = clocks.stop() if clocks is not None else None
    ms_step = statistics.median(step_runs) / K

    # ---- per-call times: the attention call and the acceptance each from a
    # graph of K back-to-back calls (median of n_rep replays); the attention
    # call's kernels apportioned by timing markers recorded inside a graph
    g_attn = capture(K, 0, lambda r, i: attn(r))
    g_acc = capture(K, 0, lambda r, i: accept(r))
    attn_ms = timer.median_ms([g_attn], n_rep) / K
    acc_ms = timer.median_ms([g_acc], n_rep) / K
    attn_names = [H.hpd_branch_attn_kernel_name(argsets[0], k) for k in range(n_launch)]
    S_mark = min(K, 50)
    events = [[torch.cuda.Event(enable_timing=True) for _ in range(n_launch + 1)]
              for _ in range(S_mark)]
    with torch.cuda.stream(stream):
        for row in events:
            for e in row:
                e.record(stream)  # creates the handle
    stream.synchronize()
    handles = [[int(e.cuda_event) for e in row] for row in events]
    g_mark = capture(S_mark, 0, lambda r, i: attn(r, handles[i]))
    with torch.cuda.stream(stream):
        g_mark.replay()
    torch.cuda.synchronize(dev)
    span = [statistics.mean(ev[k].elapsed_time(ev[k + 1]) for ev in events)
            for k in range(n_launch)]
    kernel_ms = {nm: attn_ms * span[k] / sum(span) for k, nm in enumerate(attn_names)}
    kernel_ms[ACCEPT] = acc_ms

    # ---- cold L2: before each step (and before each attention call alone) a
    # write of twice the L2 size evicts everything; events around the call
    flush = torch.empty(2 * l2, dtype=torch.uint8, device=dev)
    n_cold = max(5, min(20, K))
    ev_cold = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(n_cold)]
    torch.cuda.synchronize(dev)
    with torch.cuda.stream(stream):
        for i, (e0, e1, e2, e3) in enumerate(ev_cold):
            flush.fill_(i & 0xff)
            e0.record(stream)
            step(i % R)
            e1.record(stream)
            flush.fill_((i + 1) & 0xff)
            e2.record(stream)
            attn(i % R)
            e3.record(stream)
    torch.cuda.synchronize(dev)
    cold_step_ms = statistics.median(e0.elapsed_time(e1) for e0, e1, _, _ in ev_cold)
    cold_attn_ms = statistics.median(e2.elapsed_time(e3) for _, _, e2, e3 in ev_cold)
    del flush

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

    def e2e_capture(nsteps):
        g = torch.cuda.CUDAGraph()
        events = []  # keep the events alive with the graph
        with torch.cuda.graph(g, stream=stream):
            h2d_s.wait_stream(stream)
            d2h_s.wait_stream(stream)
            comp, out_done = {}, {}
            for i in range(nsteps):
                s_i, r = i % 2, i % R
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
                H.hpd_decode_step(slot_args(s_i, r), sl["lg"].data_ptr(), sl["dr"].data_ptr(),
                                  VOCAB, sl["tok"].data_ptr(), sl["acc"].data_ptr(), sh)
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
    ge = e2e_capture(K)
    with torch.cuda.stream(stream):
        ge.replay()  # untimed first replay
    torch.cuda.synchronize(dev)
    e2e_ms = statistics.median(timer.replay_ms([ge], sync_ranks=True) for _ in range(n_rep))
    err = op.errors(stream)
    if err:
        raise SystemExit(f"bench.py: device error flags {err:#x} on {name}")
    # the results that came back are the library's (the last replayed step's slot)
    if not torch.equal(host_out, slots[(K - 1) % 2]["dout"].cpu()):
        raise SystemExit("bench.py: end-to-end results differ from the device copy")

    # ---- numbers
    qtok = inp.B * inp.m
    pk = peaks()
    per, step_work = algorithmic_work(inp)
    dom = max(kernel_ms, key=kernel_ms.get)
    dom_ms = kernel_ms[dom]
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
    roof["traffic"] = ncu_traffic(name, dom)
    roof["kernel"] = dom
    roof["kernel_us"] = dom_ms * 1e3
    roof["algorithmic"] = {"bytes": per[dom]["bytes"], "flops": per[dom]["flops"]}
    roof["peak_source"] = pk["source"] + (" sustained bf16" if roof["bound"] == "tensor"
                                          else " HBM copy")
    roof["nominal_peak"] = NOMINAL_BF16_TFLOPS if roof["bound"] == "tensor" else NOMINAL_HBM_GBS
    roof["frac_of_nominal"] = roof["achieved"] / roof["nominal_peak"]
    # the attention call's algorithmic work, whichever kernels carry it
    attn_work = per["branch_attn_tc"]
    t_attn_roof = max(attn_work["bytes"] / (pk["hbm"] * 1e9),
                      attn_work["flops"] / (pk["tc_sustained"] * 1e12))
    t_step_roof = max(step_work["bytes"] / (pk["hbm"] * 1e9),
                      step_work["flops"] / (pk["tc_sustained"] * 1e12))
    acc_us = kernel_ms[ACCEPT] * 1e3
    res = {
        "name": name, "inp": inp, "logits_np": logits_np, "drafts_np": drafts_np,
        "value": whole_job_value(world, qtok, ms_step),
        "ms_per_step": ms_step,
        "step_replays_ms": step_runs,
        "wall_ms": wall_ms,
        "clocks": clk,
        "n_launch": n_launch,
        "roofline": roof,
        "attention_only": {
            "value": whole_job_value(world, qtok, attn_ms),
            "unit": UNIT,
            "us_per_call": attn_ms * 1e3,
            "launches": n_launch,
            "kernels": attn_names,
            "roofline_us": t_attn_roof * 1e6,
            "frac": t_attn_roof / (attn_ms * 1e-3),
            "bound": "tensor" if attn_work["flops"] / (pk["tc_sustained"] * 1e12)
                     > attn_work["bytes"] / (pk["hbm"] * 1e9) else "hbm",
            "note": "hpd_branch_attn alone (no acceptance): algorithmic time at the measured "
                    "peaks / measured call time",
        },
        "step_roofline": {"bytes": step_work["bytes"], "flops": step_work["flops"],
                          "t_roofline_us": t_step_roof * 1e6,
                          "frac": t_step_roof / (ms_step * 1e-3)},
        "kernel_us": {k: v * 1e3 for k, v in kernel_ms.items()},
        "accept_beside_attention": H.hpd_decode_step_concurrent(argsets[0]) == 1,
        "accept": {"us_per_call": acc_us, "bytes": per[ACCEPT]["bytes"],
                   "achieved_gbs": per[ACCEPT]["bytes"] / (acc_us * 1e-6) / 1e9,
                   "frac_of_measured_hbm":
                       per[ACCEPT]["bytes"] / (acc_us * 1e-6) / 1e9 / pk["hbm"],
                   "note": "greedy acceptance, HBM-bound: logits read once"},
        "cold_l2": {"step_us": cold_step_ms * 1e3, "attention_us": cold_attn_ms * 1e3,
                    "value": whole_job_value(world, qtok, cold_step_ms),
                    "note": f"median of {n_cold} single steps, each right after a write of "
                            f"{2 * l2 / 2**20:.0f} MiB (2x L2) evicted the cache"},
        "e2e": {"value": whole_job_value(world, qtok, e2e_ms / K), "unit": UNIT,
                "h2d_bytes_per_step": h2d_bytes, "d2h_bytes_per_step": d2h_bytes,
                "ms_per_step": e2e_ms / K,
                "note": "every step: q, page table, lengths, offsets, logits and drafts H2D "
                        "from pinned host memory in one packed copy, out, lse, tokens and "
                        "accepted lengths D2H in one packed copy; two slots on H2D / compute "
                        "/ D2H streams overlap a step's copies with the neighbouring steps' "
                        "kernels; prefix KV and paged KV cache resident; median of "
                        f"{n_rep} replays of a {K}-step graph"},
        "l2": f"{R} rotating input replicas ({R * rep_bytes / 2**20:.0f} MiB > 3x L2 "
              f"{l2 / 2**20:.0f} MiB)",
    }
    if not headline:
        return res

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
    g_kv = capture(K, 0, kv_pair)
    kv_ms = timer.median_ms([g_kv], n_rep) / K
    if kv.errors(stream):
        raise SystemExit(f"bench.py: KV append / rollback error flags {kv.errors(stream):#x}")
    kv_bytes = 2 * 2 * inp.B * inp.m * inp.H_kv * inp.D * 2  # K and V rows read + written
    res["kv_append_rollback"] = {
        "us_per_pair": kv_ms * 1e3, "launches_per_pair": 3, "bytes": kv_bytes,
        "achieved_gbs": kv_bytes / (kv_ms * 1e-3) / 1e9,
        "note": "hpd_kv_append (m rows per branch) + hpd_kv_rollback (all rolled back) "
                "on a pool of the workload's lengths; not part of the step metric"}

    # ---- fork detection / child branches after the acceptance (reported beside
    # the step): the step's argmax tokens, each page's first branch its layout
    # branch, with the fork token emitted at its first position (always within
    # the emitted span) and at its last emitted position
    acc_np = acc.cpu().numpy()
    fork_id = VOCAB - 1
    fork_tok = np.where(argmax_np == fork_id, 0, argmax_np).astype(np.int32)
    is_layout = np.zeros(inp.B, np.int32)
    firsts = inp.branch_cu[:-1][np.diff(inp.branch_cu) > 0]
    is_layout[firsts] = 1
    for b in firsts:
        fork_tok[b, 0] = fork_id
        fork_tok[b, min(max(int(acc_np[b]), 0), inp.m - 1)] = fork_id
    layout_pos = (inp.branch_prefix_len if inp.branch_prefix_len is not None
                  else np.repeat(np.diff(inp.prefix_cu), np.diff(inp.branch_cu))).astype(np.int32)
    layout_pos = np.maximum(layout_pos - inp.m, 0).astype(np.int32)
    f_in = [tdev(a) for a in (fork_tok, acc_np, is_layout, layout_pos, inp.branch_cu,
                               inp.branch_len, inp.page_table)]
    f_cap = inp.B * (inp.m + 1)
    f_state = {}

    def fork_call(r, i):
        f_state["out"] = H.fork_children(f_in[0], f_in[1], f_in[2], f_in[3], fork_id, f_in[4],
                                         None, f_in[5], f_in[6], f_cap, stream)

    with torch.cuda.stream(stream):
        fork_call(0, 0)
    torch.cuda.synchronize(dev)
    n_children = int(f_state["out"]["new_B"].item()) - inp.B
    g_fork = capture(K, 0, fork_call)
    fork_ms = timer.median_ms([g_fork], n_rep) / K
    res["fork_children"] = {
        "us_per_call": fork_ms * 1e3, "children": n_children,
        # one launch up to B + n_docs = 11,998 (the shared-memory scan), two beyond
        "launches": 1 if inp.B + inp.n_docs <= 11998 else 2,
        "note": "hpd_fork_children over the step's branches: every page's layout branch "
                "emits the fork token at its first and at its last emitted position; not "
                "part of the step metric"}

    # ---- the attention call on other layouts of the prefix and on the
    # layout-branch workload (reported beside the step; one input replica)
    def attn_call_us(inp_x):
        op_x = H.BranchAttn(H.DeviceInputs.from_host(inp_x), stream)
        with torch.cuda.stream(stream):
            for _ in range(3):
                op_x(stream)
        torch.cuda.synchronize(dev)
        g_x = capture(K, 0, lambda r, i: op_x(stream))
        ms = timer.median_ms([g_x], n_rep) / K
        if op_x.errors(stream):
            raise SystemExit(f"bench.py: error flags {op_x.errors(stream):#x} on {inp_x.name}")
        return ms * 1e3, H.hpd_branch_attn_launches(op_x.args)

    runs_us, _ = attn_call_us(W.page_the_prefix(inp, seed=7000 + cid, runs=True))
    scat_us, _ = attn_call_us(W.page_the_prefix(inp, seed=7000 + cid, runs=False))
    res["paged_prefix"] = {
        "us_per_call_consecutive_pages": runs_us, "us_per_call_scattered_pages": scat_us,
        "contiguous_us_per_call": attn_ms * 1e3,
        "note": "the same attention call with every page's prefix in the 16-token KV "
                "pool through a prefix page table: in consecutive pool pages (one "
                "prefill allocation) or scattered; one L2-warm input replica"}
    lay = W.make_layout_config()
    lay_us, lay_launch = attn_call_us(lay)
    res["layout_branches"] = {
        "workload": "8 pages, vision U[1024,3072], layout tokens U[64,512], each "
                    "page's layout branch + U[4,24] content branches forked after "
                    "a layout token (lognormal histories), m=4, Hq16/Hkv2, D128, "
                    "paged prefix shared with the layout branch",
        "us_per_call": lay_us, "launches": lay_launch,
        "query_tokens_per_s": lay.B * lay.m / (lay_us * 1e-6),
        "note": "attention call only, one L2-warm input replica"}
    return res


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
    stream = torch.cuda.Stream(device=dev)

    head = measure_workload(args.workload, args, world, rank, dev, stream, H, headline=True)
    others = [w for w in (args.also.split(",") if args.also else []) if w and w != args.workload]
    per_config = {}
    for w in others:
        r = measure_workload(w, args, world, rank, dev, stream, H, headline=False)
        per_config[w] = {
            "config": step_config(w, world),
            "value": r["value"], "ms_per_step": r["ms_per_step"], "roofline": r["roofline"],
            "attention_only": r["attention_only"], "step_roofline": r["step_roofline"],
            "e2e": r["e2e"], "kernel_us": r["kernel_us"], "cold_l2": r["cold_l2"],
            "accept_beside_attention": r["accept_beside_attention"],
        }
        del r
        torch.cuda.empty_cache()

    # ---- CPU baseline: the oracle on this host's cores (rank 0, N = 1 only)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        v, thr, sample = oracle_sample_run(head["inp"], head["logits_np"], head["drafts_np"],
                                           args.cpu_seconds)
        cpu = {"value": v, "unit": UNIT, "cores": thr, "kind": "oracle", "sample": sample}

    if world > 1:
        dist.destroy_process_group()
    if rank != 0:
        return None

    K = args.steps
    line = {
        "metric": METRIC, "value": head["value"], "unit": UNIT, "n_gpus": world, "steps": K,
        "warmup": max(args.warmup, 3), "ms_per_step": head["ms_per_step"],
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic",
        "config": step_config(args.workload, world),
        "timing": {
            "method": f"one CUDA graph of exactly {K} steps on the launch stream, replayed "
                      f"{len(head['step_replays_ms'])} times, each replay bracketed by a "
                      "barrier and a device synchronize and timed with CUDA events; "
                      "ms_per_step = median replay / steps",
            "replays_ms": head["step_replays_ms"],
            "l2": head["l2"],
            "per_kernel": "from graphs of back-to-back calls of each entry point after the "
                          "timed region (median of the same number of replays); the attention "
                          "call's kernels apportioned by in-graph timing markers",
        },
        "e2e": head["e2e"],
        "gpu_launches": K * (head["n_launch"] + 1),
        "roofline": head["roofline"],
        "attention_only": head["attention_only"],
        "step_roofline": head["step_roofline"],
        "kernel_us": head["kernel_us"],
        "accept": head["accept"],
        "cold_l2": head["cold_l2"],
        "accept_beside_attention": head["accept_beside_attention"],
        "per_config": per_config,
        "kv_append_rollback": head["kv_append_rollback"],
        "fork_children": head["fork_children"],
        "paged_prefix": head["paged_prefix"],
        "layout_branches": head["layout_branches"],
        "context": PAPER_CONTEXT,
        "host_wall_ms_per_step": head["wall_ms"] / K,
        "cpu_baseline": cpu,
        "clocks": head["clocks"],
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
        "config": step_config(args.workload, world),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--workload", choices=W.CONFIG_NAMES, default="c4",
                    help="the headline workload (default: c4, the largest single-GPU preset)")
    ap.add_argument("--also", default="c2,c3,c5",
                    help="comma-separated workloads measured after the headline (per_config)")
    ap.add_argument("--replays", type=int, default=5,
                    help="timed replays of the K-step graph (the median is reported; >= 5)")
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
