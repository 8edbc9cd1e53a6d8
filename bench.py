#!/usr/bin/env python
"""Benchmark of the draft-attention hot path (one drafting step per "step").

A step drafts every level of one workload's draft chain/tree: per level, the
new nodes' q/k/v are RoPE'd and appended, then they attend over
[target prefix | draft KV] (kvshot_draft_append + kvshot_draft_attn, three
kernels).  The default workload is the long-context multi-layer one (4
sequences x 4 reused target layers = 16 caches of 32768 tokens, paged P=64,
32-node depth-8 tree), the largest configuration; --workload selects another.

Printed (rank 0, one JSON line): draft tokens/s (a token attending several
reused layers counts once) over the timed steps with inputs resident in HBM,
the achieved HBM bandwidth of the draft-attention call measured live with
CUDA events (algorithmic bytes / time), the end-to-end rate through the C ABI
with host buffers, the CPU oracle's rate on a bounded sample, GPU clocks.

Multi-GPU: one process per GPU under torchrun runs an independent replica
(the path has no exchange step); value = all ranks' tokens / max time.
"""
from __future__ import annotations

import argparse
import csv
import hashlib
import io
import json
import math
import os
import re
import statistics
import subprocess
import sys
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2604_26412_gb300 import replicas  # noqa: E402
from paper_2604_26412_gb300 import workloads as wl  # noqa: E402

METRIC = "draft-attn tokens/s and achieved HBM GB/s (fraction of GB300 peak) at 1 GPU"
UNIT = "tokens/s"
FALLBACK_HBM_GBS = 6800.0


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=400)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--part", choices=["attn", "fusion", "project"], default="attn",
                    help="attn: the draft-attention step (default); fusion: the hybrid drafter's gated-delta "
                         "fusion at the hybrid-tree workload's per-depth token counts; project: the KV-only "
                         "drafter's multi-layer KV projection + RoPE fix for one step's verified tokens")
    ap.add_argument("--workload", type=int, default=5, choices=[1, 2, 3, 4, 5])
    ap.add_argument("--mode", choices=["per_depth", "whole"], default="per_depth")
    ap.add_argument("--kernel", choices=["auto", "cc", "mma", "tc"], default="auto")
    ap.add_argument("--qk-norm", action="store_true",
                    help="the append normalises q and k per head before RoPE (kvshot_draft_append_qknorm)")
    ap.add_argument("--kv-dtype", choices=["bf16", "fp8"], default="bf16",
                    help="target cache element type: bf16, or fp8 e4m3 codes with power-of-two scales "
                         "(KVSHOT_TARGET_FP8; not in the paper)")
    ap.add_argument("--num-ctas", type=int, default=0)
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-sample-seconds", type=float, default=12.0)
    ap.add_argument("--no-graph", action="store_true")
    ap.add_argument("--max-prefix", type=int, default=0,
                    help="cap every prefix length (profiling-sized cases; the default is the workload's own)")
    ap.add_argument("--page-size", type=int, default=0,
                    help="override the workload's page size (exploration; the default is the workload's own)")
    return ap.parse_args()


# ----------------------------------------------------------------- helpers

def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    elif torch.cuda.is_available():
        torch.cuda.set_device(0)
    return world, rank, local


def barrier(world):
    replicas.barrier()


def max_over_ranks(x: float, world: int) -> float:
    return replicas.max_over_ranks(x)


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return json.load(f), "measured"
    except (OSError, ValueError):
        return {"hbm_gbs": FALLBACK_HBM_GBS}, "fallback"


# Sources of the draft-attention call (the kernels whose DRAM traffic profiles/traffic.json records).
ATTN_SOURCES = ("attn_cc.cu", "attn_mma.cu", "attn_tc.cu", "kvshot_api.cu", "kvshot_attn_common.cuh",
                "kvshot_internal.h", "kvshot_tcgen05.cuh", "merge_append.cu")


# The sources each attention kernel's launches depend on: its own file, the shared producer/cursor
# header, the host planner that sizes its grid, and the merge kernel.  A traffic record names the set
# its hash covers, so an edit to one kernel leaves the other's record valid.
MMA_SOURCES = ("attn_mma.cu", "kvshot_api.cu", "kvshot_attn_common.cuh", "kvshot_internal.h", "merge_append.cu")
TC_SOURCES = ("attn_tc.cu", "kvshot_tcgen05.cuh", "kvshot_api.cu", "kvshot_attn_common.cuh", "kvshot_internal.h",
              "merge_append.cu")


# Sources of the gated-delta fusion call.
FUSION_SOURCES = ("gated_delta.cu", "kvshot_slab_gemm.cuh", "kvshot_attn_common.cuh", "kvshot_internal.h", "kvshot_tcgen05.cuh")


# Comments, string and character literals of C/C++/CUDA source, in the order a compiler reads them.
_CXX_TOKENS = re.compile(r'//[^\n]*|/\*.*?\*/|"(?:\\.|[^"\\\n])*"|\'(?:\\.|[^\'\\\n])*\'', re.S)


def code_only(text: str) -> str:
    """The source with its comments removed and its whitespace collapsed (literals kept as written)."""
    return " ".join(_CXX_TOKENS.sub(lambda m: " " if m.group(0)[0] == "/" else m.group(0), text).split())


def kernel_source_hash(sources=ATTN_SOURCES):
    """Hash of the code (comments and whitespace ignored) of the given csrc files: a traffic record
    stays valid across edits that cannot change the kernels' DRAM traffic."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2604_26412_gb300", "csrc")
    for name in sources:
        with open(os.path.join(csrc, name), encoding="utf-8") as f:
            h.update(name.encode() + b"\0" + code_only(f.read()).encode())
    return h.hexdigest()[:16]


def recorded_traffic(workload, mode, sources=ATTN_SOURCES, kernel=None):
    """DRAM bytes per call (key "w<workload>-<mode>", or "fusion-hybrid_tree") from a committed ncu
    summary, if it is for the current kernel sources (and, given `kernel`, for the attention kernel
    that ran: the record's "kernel"); else None.  The record's "sources" (default: `sources`) are the
    files its "kernel_hash" covers."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)
    except (OSError, ValueError):
        return None
    key = f"w{workload}-{mode}" if workload is not None else mode
    e = rec.get(key)
    if not e or e.get("kernel_hash") != kernel_source_hash(tuple(e.get("sources", sources))):
        return None
    if kernel is not None and e.get("kernel") != kernel:
        return None
    return e.get("dram_bytes_per_call")


def algorithmic_bytes(spec: wl.Spec, n_nodes: int, n_query: int, paged: bool, target_elem: int = 2) -> int:
    """Bytes one draft-attention call must move: K and V of every visible-key
    candidate (prefix + draft slots) once per KV head, q in, out and lse out,
    the page-table entries and lengths read.  target_elem: bytes per prefix K/V
    element (2 bf16, 1 fp8); draft K/V are bf16."""
    D = spec.head_dim
    kv = sum(spec.hkv * (L * target_elem + n_nodes * 2) * D * 2 for L in spec.seq_lens)
    qo = 2 * spec.num_caches * n_query * spec.hq * D * 2
    lse = spec.num_caches * n_query * spec.hq * 4
    pt = sum(math.ceil(L / spec.page_size) * 4 for L in spec.seq_lens) if paged else 0
    meta = spec.num_caches * 4 + (spec.num_seqs * n_nodes * 4 if spec.tree else 0)
    return kv + qo + lse + pt + meta


def algorithmic_flops(spec: wl.Spec, n_nodes: int, n_query: int) -> int:
    return sum(4 * spec.hq * n_query * (L + n_nodes) * spec.head_dim for L in spec.seq_lens)


class ClockSampler:
    """nvidia-smi clocks and throttle reasons, sampled during the timed region."""

    FIELDS = ["index", "clocks.sm", "clocks.max.sm", "power.draw", "clocks_event_reasons.active",
              "clocks_event_reasons.hw_slowdown", "clocks_event_reasons.hw_thermal_slowdown",
              "clocks_event_reasons.sw_thermal_slowdown", "clocks_event_reasons.sw_power_cap"]

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", "--query-gpu=" + ",".join(self.FIELDS), "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        rows = [r for r in csv.reader(io.StringIO(out)) if len(r) == len(self.FIELDS)]
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].strip().replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].strip().replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if v.strip().lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


# --------------------------------------------------------------- CPU oracle

def cpu_sample_spec(spec: wl.Spec) -> wl.Spec:
    """One sequence of the workload (all its reused layers), same per-cache shapes."""
    per = spec.layers
    return wl.Spec(spec.name + "-seq0", 1, spec.layers, list(spec.seq_lens[:per]), list(spec.levels), spec.tree,
                   spec.paged, page_size=spec.page_size, hq=spec.hq, hkv=spec.hkv, head_dim=spec.head_dim,
                   max_fanout=spec.max_fanout, seed=spec.seed, rope_base=spec.rope_base)


class OracleSample:
    """The CPU oracle (as it stands) on one sequence of the workload: append +
    attention of one drafting level per call."""

    def __init__(self, spec: wl.Spec, mode: str, seed: int):
        from oracle import oracle
        self.oracle = oracle
        oracle.build()
        self.spec = cpu_sample_spec(spec)
        self.inp = wl.make_inputs(self.spec, "cpu", seed=seed)
        s, inp = self.spec, self.inp
        self.tk, self.tv = wl.bf16_bits(inp.target_k), wl.bf16_bits(inp.target_v)
        self.pt = inp.page_table.numpy() if inp.page_table is not None else None
        self.lens = inp.seq_lens.numpy()
        self.par = inp.tree_parent.numpy()
        if mode == "per_depth":
            self.levels = list(s.levels)
            self.q = [wl.bf16_bits(x) for x in inp.q_in]
            self.k = [wl.bf16_bits(x) for x in inp.k_in]
            self.v = [wl.bf16_bits(x) for x in inp.v_in]
            self.pos = [x.numpy() for x in inp.positions]
        else:
            self.levels = [s.n_nodes]
            self.q = [wl.bf16_bits(torch.cat(inp.q_in, 1))]
            self.k = [wl.bf16_bits(torch.cat(inp.k_in, 1))]
            self.v = [wl.bf16_bits(torch.cat(inp.v_in, 1))]
            self.pos = [torch.cat(inp.positions, 1).numpy()]
        self.n0 = np.cumsum([0] + self.levels[:-1]).tolist()
        C, D = s.num_caches, s.head_dim
        self.dk = np.zeros((C, s.hkv, inp.n_max, D), np.uint16)
        self.dv = self.dk.copy()
        self.cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
        # fill the draft buffers once so any level can run alone
        for i in range(len(self.levels)):
            self._append(i)

    def _append(self, i):
        s, o = self.spec, self.oracle
        d = o.make_desc(num_caches=s.num_caches, num_seqs=1, hq=s.hq, hkv=s.hkv, head_dim=s.head_dim, n_nodes=0,
                        n_query=0, n_max=self.inp.n_max, tree=s.tree, l_cap=1)
        return o.append(d, self.q[i], self.k[i], self.v[i], self.pos[i], self.n0[i], self.levels[i], s.rope_base,
                        self.dk, self.dv)

    def level(self, i) -> int:
        """Append + attention of level i; returns the draft tokens it produced."""
        s, o, inp = self.spec, self.oracle, self.inp
        q_rot = self._append(i)
        n_nodes = self.n0[i] + self.levels[i]
        if s.paged:
            d = o.make_desc(num_caches=s.num_caches, num_seqs=1, hq=s.hq, hkv=s.hkv, head_dim=s.head_dim,
                            n_nodes=n_nodes, n_query=self.levels[i], n_max=inp.n_max, tree=s.tree, paged=True,
                            page_size=s.page_size, max_pages_per_seq=self.pt.shape[1], num_pages=inp.num_pages)
        else:
            d = o.make_desc(num_caches=s.num_caches, num_seqs=1, hq=s.hq, hkv=s.hkv, head_dim=s.head_dim,
                            n_nodes=n_nodes, n_query=self.levels[i], n_max=inp.n_max, tree=s.tree, l_cap=inp.l_cap)
        o.attn(d, q_rot, self.tk, self.tv, self.pt, self.lens, self.dk, self.dv,
               np.ascontiguousarray(self.par[:, :n_nodes]), nthreads=self.cores)
        return self.levels[i]

    def timed(self, budget_s: float):
        """Run levels round-robin for about budget_s seconds; (tokens/s, description)."""
        t0 = time.perf_counter()
        tokens, calls, i = 0, 0, len(self.levels) - 1
        while True:
            tokens += self.level(i)
            calls += 1
            i = (i + 1) % len(self.levels)
            if time.perf_counter() - t0 >= budget_s:
                break
        dt = time.perf_counter() - t0
        sample = (f"{calls} drafting-level calls (append + attention) on 1 of {self.spec.num_seqs} sequence(s) "
                  f"x {self.spec.layers} reused layer(s), fp64 oracle, {dt:.1f} s")
        return tokens / dt, sample, dt


# ---------------------------------------------------------------- our arm

def attn_config(spec: wl.Spec, args, world: int, bytes_per_call: float) -> dict:
    """The workload block of the JSON line; the reference arm prints the same block."""
    paged = spec.paged
    fp8 = args.kv_dtype == "fp8"
    return {
        "workload": spec.name,
        "mode": args.mode,
        "num_seqs": spec.num_seqs,
        "reused_layers": spec.layers,
        "num_caches": spec.num_caches,
        "prefix_lens": "ragged U[512,8192]" if args.workload == 4 else spec.seq_lens[0],
        "draft_levels": list(spec.levels),
        "tree": spec.tree,
        "layout": f"paged P={spec.page_size}" if paged else "contiguous",
        "target_cache": "fp8 e4m3" if fp8 else "bf16",
        "append": "QK-norm + RoPE" if args.qk_norm else "RoPE",
        "gqa": f"{spec.hq}/{spec.hkv}",
        "head_dim": spec.head_dim,
        "tokens_per_step": spec.num_seqs * spec.n_nodes,
        "l2": "inputs larger than L2 (no flush)" if bytes_per_call > 2 * 129e6
              else "inputs smaller than L2 (not flushed: latency-bound workload)",
        "parallelism": f"replicas x{world}",
    }


def mode_levels(spec: wl.Spec, mode: str):
    """Query nodes per draft-attention call of one step: one call per depth, or one for the whole tree."""
    return list(spec.levels) if mode == "per_depth" else [spec.n_nodes]


def roofline_bytes(spec: wl.Spec, levels, paged: bool, fp8: bool):
    n0s = np.cumsum([0] + list(levels)[:-1]).tolist()
    return [algorithmic_bytes(spec, n0s[i] + levels[i], levels[i], paged, 1 if fp8 else 2) for i in range(len(levels))]


def call_roofline(step, inp, spec: wl.Spec, stream, ms_per_step: float, hbm_peak: float, peak_src: str,
                  traffic_key=None, target_elem: int = 2) -> dict:
    """Live roofline of the draft-attention calls of one step (attention + merge kernels): CUDA events
    around every call on the launching stream, the stream kept busy by a sleep kernel while the host
    enqueues them; achieved = algorithmic bytes / mean call time.  traffic_key: (workload, mode) of
    the committed traffic record for this exact configuration, or None; the record is used only if
    one attention kernel ran and it is the record's."""
    from paper_2604_26412_gb300 import kvshot
    levels = step.levels
    n0s = np.cumsum([0] + levels[:-1]).tolist()
    paged = inp.page_table is not None
    reps = max(3, min(50, int(2000 / max(ms_per_step, 1e-3) / len(levels))))
    ev = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in levels]
          for _ in range(reps)]
    with torch.cuda.stream(stream):
        torch.cuda._sleep(int(2e7))  # keep the GPU busy while the host enqueues the calls
        for r in range(reps):
            for i in range(len(levels)):
                ev[r][i][0].record(stream)
                kvshot.draft_attn(step.descs[i], step.q_rot[i], step.target_k, step.target_v, inp.page_table,
                                  inp.seq_lens, step.draft_k, step.draft_v, step.parents[i], step.out[i], step.lse[i],
                                  stream)
                ev[r][i][1].record(stream)
    torch.cuda.synchronize()
    if step.error_code() != 0:
        raise RuntimeError(f"device error {step.error_code()}")
    call_ms = [statistics.mean(ev[r][i][0].elapsed_time(ev[r][i][1]) for r in range(reps)) for i in range(len(levels))]
    call_bytes = [algorithmic_bytes(spec, n0s[i] + levels[i], levels[i], paged, target_elem) for i in range(len(levels))]
    call_flops = [algorithmic_flops(spec, n0s[i] + levels[i], levels[i]) for i in range(len(levels))]
    achieved_gbs = sum(call_bytes) / (sum(call_ms) / 1e3) / 1e9
    achieved_tflops = sum(call_flops) / (sum(call_ms) / 1e3) / 1e12
    G = spec.hq // spec.hkv
    flags = step.descs[0].flags
    if flags & kvshot.KVSHOT_FORCE_CC:
        kernels = ["cuda-core"]
    elif flags & kvshot.KVSHOT_FORCE_TC:
        kernels = ["tcgen05"]
    elif flags & kvshot.KVSHOT_FORCE_MMA:
        kernels = ["m16n8k16"]
    else:  # the library's automatic choice (kvshot_api.cu make_plan)
        def auto(rows):
            tc = (16 < rows <= 128) if target_elem == 1 else rows >= 16
            return "tcgen05" if tc and 128 % G == 0 else "m16n8k16"
        kernels = sorted({auto(G * lv) for lv in levels})
    traffic = None
    if traffic_key is not None and len(kernels) == 1:
        traffic = recorded_traffic(*traffic_key, kernel=kernels[0])
    return {
        "bound": "hbm",
        "kernel": "kvshot_draft_attn (attention + merge kernels)",
        "attention_kernels": kernels,
        "achieved": round(achieved_gbs, 1),
        "peak": hbm_peak,
        "unit": "GB/s",
        "frac": round(achieved_gbs / hbm_peak, 4),
        "peak_source": f"{peak_src} (MEASURED_PEAKS.json hbm_gbs)" if peak_src == "measured" else "fallback 6.8 TB/s",
        "traffic": traffic,
        "algorithmic_bytes_per_call": int(statistics.mean(call_bytes)),
        "call_us": round(statistics.mean(call_ms) * 1e3, 2),
        "per_level_us": [round(x * 1e3, 2) for x in call_ms],
        "achieved_tflops": round(achieved_tflops, 2),
        "max_rows_per_kv_head": G * max(levels),
        "calls_timed": reps * len(levels),
        "kernel_hash": kernel_source_hash(),
    }


def gate_roofline(workload: int, args, dev, hbm_peak: float, peak_src: str) -> dict:
    """Live roofline of another workload's draft-attention calls (per depth, default kernels), measured
    in the same process after a few untimed steps."""
    from paper_2604_26412_gb300.step import DraftStep
    spec = wl.config(workload, seed=args.seed)
    inp = wl.make_inputs(spec, dev, seed=args.seed)
    step = DraftStep(inp, mode="per_depth")
    stream = torch.cuda.Stream()
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        for _ in range(3):
            step.run()
    s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        s0.record(stream)
        for _ in range(5):
            step.run()
        s1.record(stream)
    torch.cuda.synchronize()
    r = call_roofline(step, inp, spec, stream, s0.elapsed_time(s1) / 5, hbm_peak, peak_src,
                      traffic_key=(workload, "per_depth"))
    out = {"workload": spec.name, "mode": "per_depth"}
    out.update({k: r[k] for k in ("frac", "achieved", "unit", "call_us", "per_level_us", "traffic",
                                  "algorithmic_bytes_per_call", "attention_kernels", "calls_timed")})
    del step, inp
    torch.cuda.empty_cache()
    return out



def run_ours(args, world, rank, local):
    from paper_2604_26412_gb300 import kvshot
    from paper_2604_26412_gb300.step import DraftStep

    dev = torch.device("cuda", torch.cuda.current_device())
    spec = wl.config(args.workload, seed=args.seed)
    if args.page_size:
        spec.page_size = args.page_size
    if args.max_prefix:
        spec.seq_lens = [min(L, args.max_prefix) for L in spec.seq_lens]
    inp = wl.make_inputs(spec, dev, seed=args.seed + 1000 * rank)
    flags = {"auto": 0, "cc": kvshot.KVSHOT_FORCE_CC, "mma": kvshot.KVSHOT_FORCE_MMA,
             "tc": kvshot.KVSHOT_FORCE_TC}[args.kernel]
    fp8 = args.kv_dtype == "fp8"
    target_fp8 = (*wl.fp8_target(inp), wl.FP8_K_EXP, wl.FP8_V_EXP) if fp8 else None
    qk_norm = None
    if args.qk_norm:  # synthetic per-dimension weights around 1, Qwen3's eps
        g = torch.Generator().manual_seed(args.seed + 17)
        qk_norm = tuple((0.5 + torch.rand(spec.head_dim, generator=g)).to(torch.bfloat16).to(dev) for _ in range(2)) \
            + (1e-6,)
    step = DraftStep(inp, mode=args.mode, flags=flags, num_ctas=args.num_ctas, target_fp8=target_fp8,
                     qk_norm=qk_norm)
    paged = inp.page_table is not None
    stream = torch.cuda.Stream()
    torch.cuda.synchronize()

    with torch.cuda.stream(stream):
        for _ in range(max(3, args.warmup)):
            step.run()
    torch.cuda.synchronize()
    if step.error_code() != 0:
        raise RuntimeError(f"device error {step.error_code()}")

    graph = None
    if not args.no_graph:
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=stream):
            step.run()
        with torch.cuda.stream(stream):
            for _ in range(2):
                graph.replay()
        torch.cuda.synchronize()

    # ---- timed region: K steps, inputs resident in HBM (larger than L2 for the long-prefix workloads)
    clocks = ClockSampler(local)
    barrier(world)
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.3)
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        t_start.record(stream)
        for _ in range(args.steps):
            if graph is not None:
                graph.replay()
            else:
                step.run()
        t_end.record(stream)
    torch.cuda.synchronize()
    clock_info = clocks.stop()
    barrier(world)
    ms_total = max_over_ranks(t_start.elapsed_time(t_end), world)
    ms_per_step = ms_total / args.steps
    tokens_per_step = step.tokens
    value = replicas.whole_job_rate(tokens_per_step, args.steps, world, ms_total)

    # ---- live roofline of the draft-attention call (attention + merge kernels), per level
    peaks, peak_src = measured_peaks()
    hbm_peak = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    # A traffic record holds for the stock workload only (no prefix cap, page size or grid override).
    stock = not args.max_prefix and not args.page_size and not args.num_ctas
    roofline = call_roofline(step, inp, spec, stream, ms_per_step, hbm_peak, peak_src,
                             traffic_key=(args.workload, args.mode + ("-fp8" if fp8 else "")) if stock else None,
                             target_elem=1 if fp8 else 2)
    gates = None
    if args.workload == 5 and args.mode == "per_depth" and not fp8 and flags == 0 and not args.qk_norm \
            and not args.max_prefix and not args.page_size:
        # The other long-prefix workloads, per depth, measured the same way in the same process.
        gate_clocks = ClockSampler(local)
        gate_clocks.start()
        gates = {f"w{w}": gate_roofline(w, args, dev, hbm_peak, peak_src) for w in (3, 4)}
        gates["clocks"] = gate_clocks.stop()
        gates["w5"] = {k: roofline[k] for k in ("frac", "achieved", "call_us")}

    # ---- end to end through the C ABI with host buffers (pinned), copies in the timed region
    e2e = run_e2e(args, step, inp, stream, world)

    gpu_launches = 3 * len(step.levels) * args.steps
    result = {
        "metric": METRIC,
        "value": round(value, 1),
        "unit": UNIT,
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(ms_per_step, 5),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16 (target K/V fp8 e4m3)" if fp8 else "bf16",
        "data": "synthetic (seeded N(0,1) K/V, N(0,1)/sqrt(128) q; shapes of the paper's Qwen3-8B runs)"
                + (f"; target cache as e4m3 codes x 2^{wl.FP8_K_EXP} (K), 2^{wl.FP8_V_EXP} (V)" if fp8 else ""),
        "config": attn_config(spec, args, world, sum(roofline_bytes(spec, step.levels, paged, fp8)) / len(step.levels)),
        "cuda_graph": graph is not None,
        "roofline": roofline,
        "e2e": e2e,
        "clocks": clock_info,
        "gpu_launches": gpu_launches,
    }
    if gates is not None:
        result["gates"] = gates
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        samp = OracleSample(spec, args.mode, args.seed)
        v, desc, _ = samp.timed(args.cpu_sample_seconds)
        result["cpu_baseline"] = {"value": round(v, 3), "unit": UNIT, "cores": samp.cores, "kind": "oracle",
                                  "sample": desc}
    return result


FUSION_METRIC = "gated-delta fusion tokens/s and achieved HBM GB/s (fraction of GB300 peak) at 1 GPU"


def fusion_bytes(T: int, d: int) -> int:
    """Algorithmic bytes of one fusion call: W_g and W_delta (4 d^2 bf16), b_g, n, o and h."""
    return 2 * (4 * d * d + d + 3 * T * d)


class FusionOracleSample:
    """The fusion oracle (as it stands) on one level's tokens."""

    def __init__(self, fi, T):
        from oracle import fusion as fo
        self.fo = fo
        self.T = T
        self.args = [wl.bf16_bits(x.cpu()) for x in (fi.n[:T], fi.o[:T], fi.w_g, fi.b_g, fi.w_delta)]
        self.cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()

    def timed(self, budget_s: float):
        t0, calls = time.perf_counter(), 0
        while True:
            self.fo.gated_delta(*self.args)
            calls += 1
            if time.perf_counter() - t0 >= budget_s:
                break
        dt = time.perf_counter() - t0
        return self.T * calls / dt, f"{calls} fusion calls of {self.T} tokens x d={self.args[0].shape[1]}, fp64 " \
            f"oracle (numpy matrix products), {dt:.1f} s", dt


def run_fusion(args, world, rank, local):
    """The hybrid drafter's gated-delta fusion (Sec. 3.4) for the hybrid-tree workload: one call per
    drafting depth on the tokens of that depth (sequences x level size), hidden size d = 4096."""
    from paper_2604_26412_gb300 import kvshot
    spec = wl.config(3, seed=args.seed)
    d = wl.HIDDEN
    tokens = [spec.num_seqs * lv for lv in spec.levels]
    T_max = max(tokens)
    fi = wl.fusion_inputs(T_max, d, device="cuda", seed=args.seed + 5)
    stream = torch.cuda.Stream()
    descs, outs = [], []
    ws_bytes = max(kvshot.gated_delta_workspace_size(kvshot.make_fusion_desc(num_tokens=T, hidden=d)) for T in tokens)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    for T in tokens:
        descs.append(kvshot.make_fusion_desc(num_tokens=T, hidden=d, workspace=ws, workspace_bytes=ws_bytes,
                                             err_flag=err))
        outs.append(torch.empty((T, d), dtype=torch.bfloat16, device="cuda"))

    def step():
        for i, T in enumerate(tokens):
            kvshot.gated_delta(descs[i], fi.n[:T], fi.o[:T], fi.w_g, fi.b_g, fi.w_delta, outs[i], stream)

    with torch.cuda.stream(stream):
        for _ in range(max(3, args.warmup)):
            step()
    torch.cuda.synchronize()
    graph = None
    if not args.no_graph:
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=stream):
            step()
        torch.cuda.synchronize()
    run = (lambda: graph.replay()) if graph is not None else step
    clocks = ClockSampler(local)
    barrier(world)
    torch.cuda.synchronize()
    clocks.start()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        t0.record(stream)
        for _ in range(args.steps):
            run()
        t1.record(stream)
    torch.cuda.synchronize()
    clock_info = clocks.stop()
    barrier(world)
    ms_total = max_over_ranks(t0.elapsed_time(t1), world)
    ms_per_step = ms_total / args.steps
    value = replicas.whole_job_rate(sum(tokens), args.steps, world, ms_total)
    assert int(err.item()) == 0, f"device error {int(err.item())}"

    # live roofline: CUDA events around every call on the launching stream
    reps = 30
    ev = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in tokens]
          for _ in range(reps)]
    with torch.cuda.stream(stream):
        torch.cuda._sleep(int(2e7))
        for r in range(reps):
            for i, T in enumerate(tokens):
                ev[r][i][0].record(stream)
                kvshot.gated_delta(descs[i], fi.n[:T], fi.o[:T], fi.w_g, fi.b_g, fi.w_delta, outs[i], stream)
                ev[r][i][1].record(stream)
    torch.cuda.synchronize()
    call_ms = [statistics.mean(ev[r][i][0].elapsed_time(ev[r][i][1]) for r in range(reps)) for i in range(len(tokens))]
    call_bytes = [fusion_bytes(T, d) for T in tokens]
    call_flops = [8 * T * d * d for T in tokens]
    achieved = sum(call_bytes) / (sum(call_ms) / 1e3) / 1e9
    peaks, peak_src = measured_peaks()
    hbm_peak = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    roofline = {
        "bound": "hbm",
        "kernel": "kvshot_gated_delta (tcgen05 GEMM + gate kernels)",
        "achieved": round(achieved, 1),
        "peak": hbm_peak,
        "unit": "GB/s",
        "frac": round(achieved / hbm_peak, 4),
        "peak_source": f"{peak_src} (MEASURED_PEAKS.json hbm_gbs)" if peak_src == "measured" else "fallback 6.8 TB/s",
        "traffic": recorded_traffic(None, "fusion-hybrid_tree", FUSION_SOURCES),
        "algorithmic_bytes_per_call": int(statistics.mean(call_bytes)),
        "call_us": round(statistics.mean(call_ms) * 1e3, 2),
        "per_level_us": [round(x * 1e3, 2) for x in call_ms],
        "achieved_tflops": round(sum(call_flops) / (sum(call_ms) / 1e3) / 1e12, 2),
        "kernel_hash": kernel_source_hash(FUSION_SOURCES),
    }

    # end to end: the branches copied in from pinned host memory and h copied back every step
    n_h = fi.n.cpu().pin_memory()
    o_h = fi.o.cpu().pin_memory()
    h_h = [torch.empty((T, d), dtype=torch.bfloat16).pin_memory() for T in tokens]
    n_d, o_d = torch.empty_like(fi.n), torch.empty_like(fi.o)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e2e_steps = max(3, min(args.steps, 50))
    with torch.cuda.stream(stream):
        e0.record(stream)
        for _ in range(e2e_steps):
            n_d.copy_(n_h, non_blocking=True)
            o_d.copy_(o_h, non_blocking=True)
            for i, T in enumerate(tokens):
                kvshot.gated_delta(descs[i], n_d[:T], o_d[:T], fi.w_g, fi.b_g, fi.w_delta, outs[i], stream)
                h_h[i].copy_(outs[i], non_blocking=True)
        e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1), world)
    e2e = {"value": round(replicas.whole_job_rate(sum(tokens), e2e_steps, world, e2e_ms), 1), "unit": UNIT,
           "h2d_bytes_per_step": 2 * T_max * d * 2, "d2h_bytes_per_step": sum(tokens) * d * 2}

    result = {
        "metric": FUSION_METRIC,
        "value": round(value, 1),
        "unit": UNIT,
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(ms_per_step, 5),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) branches, N(0,1/(3d)) W_g, N(0,1/d) W_delta; no trained weights)",
        "config": {
            "workload": "hybrid tree, gated-delta fusion step (Sec. 3.4)",
            "hidden": d,
            "tokens_per_call": tokens,
            "tokens_per_step": sum(tokens),
            "cuda_graph": graph is not None,
            "l2": "weights (134 MB per call) larger than L2 (no flush)",
            "parallelism": f"replicas x{world}",
        },
        "roofline": roofline,
        "e2e": e2e,
        "clocks": clock_info,
        "gpu_launches": 2 * len(tokens) * args.steps,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        samp = FusionOracleSample(fi, tokens[len(tokens) // 2])
        v, desc, _ = samp.timed(args.cpu_sample_seconds)
        result["cpu_baseline"] = {"value": round(v, 3), "unit": UNIT, "cores": samp.cores, "kind": "oracle",
                                  "sample": desc}
    return result


PROJECT_METRIC = "multi-layer KV projection tokens/s and achieved HBM GB/s (fraction of GB300 peak) at 1 GPU"


def project_bytes(T: int, L: int, dkv: int) -> int:
    """Algorithmic bytes of one projection call: W_K, W_V, the tokens' L-layer K/V in, their K'/V' out."""
    return 2 * (2 * dkv * L * dkv + 2 * T * L * dkv + 2 * T * dkv)


def run_project(args, world, rank, local):
    """The KV-only drafter's linear projection with RoPE fix (Sec. 3.2) on the multi-layer workload's
    shape: 4 sequences x 4 sampled target layers, 8 KV heads, paged P = 64; one call per decoding step
    projects the step's verified tokens (here 8 per sequence, a full chain accepted) into the reused cache."""
    from paper_2604_26412_gb300 import kvshot
    spec = wl.config(5, seed=args.seed)
    L, hkv, P = spec.layers, spec.hkv, spec.page_size
    B, per_seq = spec.num_seqs, 8  # tokens verified per sequence this step (a full chain of 8 accepted)
    T = B * per_seq
    dkv = hkv * wl.HEAD_DIM
    pi = wl.project_inputs(T, L, hkv, device="cuda", seed=args.seed + 7)
    cap = 4096
    pages_per = cap // P
    rng = np.random.default_rng(args.seed)
    num_pages = B * pages_per
    page_table = torch.from_numpy(rng.permutation(num_pages).reshape(B, pages_per).astype(np.int32)).cuda()
    token_cache = torch.arange(B, dtype=torch.int32, device="cuda").repeat_interleave(per_seq)
    positions = (torch.arange(per_seq, dtype=torch.int32, device="cuda") + 3000).repeat(B)
    k_pool = torch.zeros((num_pages * hkv * P, wl.HEAD_DIM), dtype=torch.bfloat16, device="cuda")
    v_pool = torch.zeros_like(k_pool)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    desc = kvshot.make_project_desc(num_tokens=T, num_layers=L, hkv=hkv, num_caches=B, page_size=P,
                                    max_pages_per_seq=pages_per, num_pages=num_pages, rope_base=spec.rope_base,
                                    rope=True, err_flag=err)
    ws = torch.empty(kvshot.kv_project_workspace_size(desc), dtype=torch.uint8, device="cuda")
    desc.workspace, desc.workspace_bytes = ws.data_ptr(), ws.numel()
    stream = torch.cuda.Stream()
    call = lambda k_in, v_in: kvshot.kv_project(desc, k_in, v_in, pi.w_k, pi.w_v, token_cache, positions, page_table,
                                                k_pool, v_pool, stream)
    with torch.cuda.stream(stream):
        for _ in range(max(3, args.warmup)):
            call(pi.k_in, pi.v_in)
    torch.cuda.synchronize()
    graph = None
    if not args.no_graph:
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=stream):
            call(pi.k_in, pi.v_in)
        torch.cuda.synchronize()
    run = (lambda: graph.replay()) if graph is not None else (lambda: call(pi.k_in, pi.v_in))
    clocks = ClockSampler(local)
    barrier(world)
    torch.cuda.synchronize()
    clocks.start()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        t0.record(stream)
        for _ in range(args.steps):
            run()
        t1.record(stream)
    torch.cuda.synchronize()
    clock_info = clocks.stop()
    barrier(world)
    ms_total = max_over_ranks(t0.elapsed_time(t1), world)
    assert int(err.item()) == 0, f"device error {int(err.item())}"
    reps = 50
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(reps)]
    with torch.cuda.stream(stream):
        torch.cuda._sleep(int(2e7))
        for a, b in ev:
            a.record(stream)
            call(pi.k_in, pi.v_in)
            b.record(stream)
    torch.cuda.synchronize()
    call_ms = statistics.mean(a.elapsed_time(b) for a, b in ev)
    # Launch floor: the same two-kernel call on 1 token, 1 layer and 1 KV head (fixed costs only).
    fl_in = wl.project_inputs(1, 1, 1, device="cuda", seed=args.seed + 9)
    fl_pool = torch.zeros((P, wl.HEAD_DIM), dtype=torch.bfloat16, device="cuda")
    fl_pt = torch.zeros((1, 1), dtype=torch.int32, device="cuda")
    fl_desc = kvshot.make_project_desc(num_tokens=1, num_layers=1, hkv=1, num_caches=1, page_size=P,
                                       max_pages_per_seq=1, num_pages=1, rope_base=spec.rope_base, rope=True,
                                       err_flag=err)
    fl_ws = torch.empty(max(256, kvshot.kv_project_workspace_size(fl_desc)), dtype=torch.uint8, device="cuda")
    fl_desc.workspace, fl_desc.workspace_bytes = fl_ws.data_ptr(), fl_ws.numel()
    fl_tc = torch.zeros(1, dtype=torch.int32, device="cuda")
    fl_v = torch.zeros_like(fl_pool)
    fl_call = lambda: kvshot.kv_project(fl_desc, fl_in.k_in, fl_in.v_in, fl_in.w_k, fl_in.w_v, fl_tc, fl_tc, fl_pt,
                                        fl_pool, fl_v, stream)
    ev_fl = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(reps)]
    with torch.cuda.stream(stream):
        for _ in range(3):
            fl_call()
        torch.cuda._sleep(int(2e7))
        for a, b in ev_fl:
            a.record(stream)
            fl_call()
            b.record(stream)
    torch.cuda.synchronize()
    floor_ms = statistics.mean(a.elapsed_time(b) for a, b in ev_fl)
    nbytes = project_bytes(T, L, dkv)
    peaks, peak_src = measured_peaks()
    hbm_peak = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    achieved = nbytes / (call_ms / 1e3) / 1e9
    roofline = {"bound": "hbm", "kernel": "kvshot_kv_project (tcgen05 slab GEMM + RoPE/store kernels)",
                "achieved": round(achieved, 1), "peak": hbm_peak, "unit": "GB/s", "frac": round(achieved / hbm_peak, 4),
                "peak_source": f"{peak_src} (MEASURED_PEAKS.json hbm_gbs)" if peak_src == "measured" else "fallback 6.8 TB/s",
                "traffic": None, "algorithmic_bytes_per_call": nbytes, "call_us": round(call_ms * 1e3, 2),
                "launch_floor_us": round(floor_ms * 1e3, 2),
                "launch_floor": "the same call on 1 token x 1 layer x 1 KV head (both kernels' fixed costs)"}
    k_h, v_h = pi.k_in.cpu().pin_memory(), pi.v_in.cpu().pin_memory()
    k_d, v_d = torch.empty_like(pi.k_in), torch.empty_like(pi.v_in)
    e2e_steps = max(3, min(args.steps, 100))
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e0.record(stream)
        for _ in range(e2e_steps):
            k_d.copy_(k_h, non_blocking=True)
            v_d.copy_(v_h, non_blocking=True)
            call(k_d, v_d)
            err_h = err.to("cpu", non_blocking=True)
        e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1), world)
    result = {
        "metric": PROJECT_METRIC, "value": round(replicas.whole_job_rate(T, args.steps, world, ms_total), 1),
        "unit": UNIT, "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(ms_total / args.steps, 5), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) K/V of the sampled layers, N(0,1/(L d_kv)) W_K, W_V; no trained weights)",
        "config": {"workload": "multi-layer KV projection + RoPE fix (Sec. 3.2)", "tokens_per_call": T,
                   "layers": L, "hkv": hkv, "layout": f"paged P={P}", "cuda_graph": graph is not None,
                   "l2": "weights and inputs (17 MB) fit in L2; no flush (launch-bound call)",
                   "parallelism": f"replicas x{world}"},
        "roofline": roofline,
        "e2e": {"value": round(replicas.whole_job_rate(T, e2e_steps, world, e2e_ms), 1), "unit": UNIT,
                "h2d_bytes_per_step": 2 * T * L * dkv * 2, "d2h_bytes_per_step": 4},
        "clocks": clock_info,
        "gpu_launches": 2 * args.steps,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        from oracle import project as po
        args_cpu = [wl.bf16_bits(x.cpu()) for x in (pi.k_in, pi.v_in, pi.w_k, pi.w_v)]
        pos_np = positions.cpu().numpy()
        t_start, calls = time.perf_counter(), 0
        while time.perf_counter() - t_start < args.cpu_sample_seconds:
            po.kv_project(*args_cpu, pos_np, spec.rope_base, True)
            calls += 1
        dt = time.perf_counter() - t_start
        cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
        result["cpu_baseline"] = {"value": round(T * calls / dt, 3), "unit": UNIT, "cores": cores, "kind": "oracle",
                                  "sample": f"{calls} projection calls of {T} tokens, fp64 oracle, {dt:.1f} s"}
    return result


def _arena(tensors, device):
    """One device buffer holding every tensor (256-byte aligned slots) and views of it shaped like
    them; returns (buffer, views, total bytes)."""
    offs, off = [], 0
    for t in tensors:
        offs.append(off)
        off += (t.numel() * t.element_size() + 255) // 256 * 256
    buf = torch.empty(max(off, 256), dtype=torch.uint8, device=device)
    views = [buf[o:o + t.numel() * t.element_size()].view(t.dtype).view(t.shape) for o, t in zip(offs, tensors)]
    return buf, views, off


def run_e2e(args, step, inp, stream, world):
    """Same steps through the C ABI, with the per-step inputs copied from pinned host memory and
    the outputs copied back inside the timed region.  A serving loop would keep a step's inputs in
    one host arena: the step's device inputs (q/k/v/positions of every level, parents, lengths,
    page table) are views of one device buffer filled by one copy per step, and its outputs
    (out and lse of every level) views of one buffer read back by one copy."""
    import dataclasses
    ins = [t for lst in (step.q_in, step.k_in, step.v_in, step.pos) for t in lst] + list(step.parents) + \
        [inp.seq_lens] + ([inp.page_table] if inp.page_table is not None else [])
    dbuf_in, views_in, h2d = _arena(ins, ins[0].device)
    for v, t in zip(views_in, ins):
        v.copy_(t)
    k = 0
    for lst in (step.q_in, step.k_in, step.v_in, step.pos):
        for i in range(len(lst)):
            lst[i] = views_in[k]
            k += 1
    for i in range(len(step.parents)):
        step.parents[i] = views_in[k]
        k += 1
    inp_e2e = dataclasses.replace(inp, seq_lens=views_in[k],
                                  page_table=views_in[k + 1] if inp.page_table is not None else None)
    inp_saved, step.inp = step.inp, inp_e2e
    outs = list(step.out) + list(step.lse)
    dbuf_out, views_out, d2h = _arena(outs, outs[0].device)
    nl = len(step.out)
    step.out = views_out[:nl]
    step.lse = views_out[nl:]
    host_in = dbuf_in.cpu().pin_memory()
    host_out = torch.empty(dbuf_out.numel(), dtype=torch.uint8).pin_memory()
    steps = max(3, min(args.steps, 100))
    with torch.cuda.stream(stream):  # one untimed pass through the new buffers
        dbuf_in.copy_(host_in, non_blocking=True)
        step.run()
    torch.cuda.synchronize()
    barrier(world)
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        a.record(stream)
        for _ in range(steps):
            dbuf_in.copy_(host_in, non_blocking=True)
            step.run()
            host_out.copy_(dbuf_out, non_blocking=True)
        b.record(stream)
    torch.cuda.synchronize()
    step.inp = inp_saved
    ms = max_over_ranks(a.elapsed_time(b), world)
    value = replicas.whole_job_rate(step.tokens, steps, world, ms)
    return {"value": round(value, 1), "unit": UNIT, "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "steps": steps, "api": "kvshot_draft_append + kvshot_draft_attn via ctypes, no CUDA graph; "
                                   "inputs and outputs in one pinned host arena each (one copy each way per step)"}


# --------------------------------------------------------- reference arm

def run_reference_fusion(args):
    """The fusion oracle as it stands on the host cores; each step is one call on the tokens of the
    hybrid-tree workload's widest drafting depth (d = 4096)."""
    spec = wl.config(3, seed=args.seed)
    T = spec.num_seqs * max(spec.levels)
    samp = FusionOracleSample(wl.fusion_inputs(T, wl.HIDDEN, device="cpu", seed=args.seed + 5), T)
    for _ in range(args.warmup):
        samp.fo.gated_delta(*samp.args)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        samp.fo.gated_delta(*samp.args)
    dt = time.perf_counter() - t0
    value = T * args.steps / dt
    return {
        "impl": "reference", "metric": FUSION_METRIC, "value": round(value, 3), "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(dt / args.steps * 1e3, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded; same shapes as the GPU arm)",
        "config": {"workload": "hybrid tree, gated-delta fusion step (Sec. 3.4)", "hidden": wl.HIDDEN,
                   "tokens_per_call": T, "parallelism": "host cores"},
        "cpu_baseline": {"value": round(value, 3), "unit": UNIT, "cores": samp.cores, "kind": "oracle",
                         "sample": f"{args.steps} fusion calls of {T} tokens, fp64 oracle"},
        "e2e": {"value": round(value, 3), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "gpu_launches": 0,
    }


def run_reference_project(args):
    """The projection oracle as it stands on the host cores; each step projects one decoding step's
    verified tokens (4 sequences x 8) of the multi-layer workload."""
    from oracle import project as po
    spec = wl.config(5, seed=args.seed)
    T = spec.num_seqs * 8
    pi = wl.project_inputs(T, spec.layers, spec.hkv, device="cpu", seed=args.seed + 7)
    a = [wl.bf16_bits(x) for x in (pi.k_in, pi.v_in, pi.w_k, pi.w_v)]
    pos = np.tile(np.arange(8) + 3000, spec.num_seqs)
    for _ in range(args.warmup):
        po.kv_project(*a, pos, spec.rope_base, True)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        po.kv_project(*a, pos, spec.rope_base, True)
    dt = time.perf_counter() - t0
    value = T * args.steps / dt
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    return {
        "impl": "reference", "metric": PROJECT_METRIC, "value": round(value, 3), "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(dt / args.steps * 1e3, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded; same shapes as the GPU arm)",
        "config": {"workload": "multi-layer KV projection + RoPE fix (Sec. 3.2)", "tokens_per_call": T,
                   "parallelism": "host cores"},
        "cpu_baseline": {"value": round(value, 3), "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": f"{args.steps} projection calls of {T} tokens, fp64 oracle"},
        "e2e": {"value": round(value, 3), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "gpu_launches": 0,
    }


def run_reference(args):
    """The CPU fp64 oracle as it stands, timed on the host cores; each step is
    one drafting level (append + attention) of one sequence of the workload."""
    if args.part == "fusion":
        return run_reference_fusion(args)
    if args.part == "project":
        return run_reference_project(args)
    spec = wl.config(args.workload, seed=args.seed)
    samp = OracleSample(spec, args.mode, args.seed)
    for w in range(args.warmup):
        samp.level(w % len(samp.levels))
    t0 = time.perf_counter()
    tokens = 0
    for k in range(args.steps):
        tokens += samp.level(k % len(samp.levels))
    dt = time.perf_counter() - t0
    value = tokens / dt
    sample = (f"{args.steps} drafting-level calls (append + attention) on 1 of {spec.num_seqs} sequence(s) x "
              f"{spec.layers} reused layer(s), fp64 oracle")
    return {
        "impl": "reference",
        "metric": METRIC,
        "value": round(value, 3),
        "unit": UNIT,
        "n_gpus": args.gpus,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(dt / args.steps * 1e3, 3),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f64",
        "data": "synthetic (seeded; same shapes as the GPU arm)",
        "config": attn_config(spec, args, args.gpus,
                              sum(roofline_bytes(spec, mode_levels(spec, args.mode), spec.paged,
                                                 args.kv_dtype == "fp8")) / len(mode_levels(spec, args.mode))),
        "host_parallelism": f"fp64 oracle on {samp.cores} host cores (rank 0 only)",
        "cpu_baseline": {"value": round(value, 3), "unit": UNIT, "cores": samp.cores, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": round(value, 3), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "gpu_launches": 0,
    }


def main():
    args = parse_args()
    if args.impl == "reference":
        rank = int(os.environ.get("RANK", "0"))
        if rank != 0:
            return
        print(json.dumps(run_reference(args)), flush=True)
        return
    world, rank, local = dist_setup()
    result = {"fusion": run_fusion, "project": run_project}.get(args.part, run_ours)(args, world, rank, local)
    if rank == 0:
        print(json.dumps(result), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
