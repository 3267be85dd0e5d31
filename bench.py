#!/usr/bin/env python3
"""Benchmark of smashed-KV decode attention (HAMburger macro-step hot path) on GB300.

One step = one macro-step of one layer for the whole batch, through the C ABI.  Default
(--path fused): ham_decode_step, which appends the macro-step's slot (RoPE of q and k at
its position) and runs split-KV attention over all slots in one pass over the cache.
--path split: ham_kv_append followed by ham_decode_attn (the same work in three kernels).
The default workload is the Llama-3-8B-shaped layer: batch 8, 32 query / 8 KV heads,
head_dim 128, 4096 slots per sequence in 16-slot pages scattered over a shared pool.

Timing: steps are captured in CUDA graphs (64 steps per graph) and replayed; the timed
region is bracketed by a barrier and a device synchronize.  Four independent caches are
rotated so each step reads a cache last touched three steps earlier (4 x 128 MiB of KV,
far above the 129 MB L2).  After each graph the four caches are rolled back to 4096 slots
(ham_kv_set_lengths), so the attended length stays 4097..4112.  The attention kernel's
own duration comes from CUDA events recorded around each of its launches inside the graph
(fused: the step's attention + combine/commit kernels; split: attention + combine).

Prints ONE JSON line on rank 0.  `--impl reference` times the CPU oracle instead.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "macro-steps/s and achieved HBM GB/s (% of GB300 peak) for smashed-KV decode attn"
UNIT = "macro-steps/s"
GRAPH_STEPS = 64
CACHES = 4
FALLBACK_HBM_GBS = 6800.0


def parse_args():
    p = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=40960)
    p.add_argument("--warmup", type=int, default=640)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", default="llama8b_layer_b8_s4096")
    p.add_argument("--e2e-steps", type=int, default=2000)
    p.add_argument("--cpu-seconds", type=float, default=12.0,
                   help="CPU work budget of the oracle baseline sample")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--min-seconds", type=float, default=1.2,
                   help="decode workloads: whole 64-step graphs are replayed until the timed "
                        "region lasts at least this long, whatever --steps asks for")
    p.add_argument("--no-target-point", action="store_true",
                   help="default workload: skip the batch 8 x 8192 slots point")
    p.add_argument("--kv", choices=["bf16", "fp8"], default="bf16",
                   help="decode workloads: bf16 pools, or FP8 (e4m3) pools with one power-of-two "
                        "scale per row")
    p.add_argument("--path", choices=["fused", "split"], default="fused",
                   help="fused: ham_decode_step; split: ham_kv_append + ham_decode_attn")
    p.add_argument("--caches", type=int, default=CACHES,
                   help="independent caches rotated by the timed steps (fewer keep an ncu capture "
                        "of a large workload within a few GB; the default keeps each step's cache "
                        "out of L2)")
    return p.parse_args()


# ---------------------------------------------------------------------------------------
# environment helpers
# ---------------------------------------------------------------------------------------

def dist_env():
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("LOCAL_RANK", "0")),
            int(os.environ.get("WORLD_SIZE", "1")))


def max_over_ranks(value, world, device):
    """The largest of every rank's `value` (the job is as slow as its slowest rank)."""
    if world == 1:
        return float(value)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(steps_per_rank, world, elapsed_s):
    """Whole-job macro-steps/s: every rank runs its own batch (weak scaling)."""
    return world * steps_per_rank / elapsed_s


def rank_cache_seed(workload_seed, rank, cache):
    """Seed of one rank's cache: ranks own different sequences."""
    return 1000 * workload_seed + 10 * rank + cache


def measured_peak_bf16(sustained=False):
    key = "bf16_tflops_sustained" if sustained else "bf16_tflops"
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)[key]), f"measured (MEASURED_PEAKS.json {key})"
    except Exception:
        return (1700.0 if sustained else 1900.0), "fallback"


def measured_peak_hbm():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["hbm_gbs"]), "measured (MEASURED_PEAKS.json hbm_gbs)"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


ATTN_SOURCES = ("ham_attn.cu", "ham_attn.cuh", "ham_internal.cuh", "ham_ptx.cuh")
ATTN_FP8_SOURCES = ("ham_attn_fp8.cu",) + ATTN_SOURCES
FRONT_SOURCES = ("ham_front.cu", "ham_front.cuh", "ham_ptx.cuh")


def kernel_source_hash(names=ATTN_SOURCES):
    """Hash of a kernel's code (comments and blank space removed), which ties an ncu summary to
    the code it measured."""
    h = hashlib.sha256()
    for name in names:
        with open(os.path.join(ROOT, "paper_2505_20438_gb300", "csrc", name)) as f:
            text = f.read()
        text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
        text = re.sub(r"//[^\n]*", " ", text)
        h.update(" ".join(text.split()).encode())
    return h.hexdigest()[:16]


def profiled_traffic(kernel, workload_name, sources=ATTN_SOURCES):
    """dram read+write bytes per launch of `kernel` (decode_step, decode_attn, front) from the
    committed ncu summary, if it was taken on the current kernel source."""
    path = os.path.join(ROOT, "profiles", f"{kernel}_{workload_name}.md")
    try:
        text = open(path).read()
    except OSError:
        return None
    src = re.search(r"kernel_source_sha256:\s*([0-9a-f]+)", text)
    tr = re.search(r"traffic_bytes_per_launch:\s*([0-9]+)", text)
    if not src or not tr or src.group(1) != kernel_source_hash(sources):
        return None
    return int(tr.group(1))


class ClockSampler:
    """nvidia-smi clocks and throttle reasons, sampled every 200 ms while running."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200", "-f", self.path],
                stdout=subprocess.DEVNULL, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.25)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        rows = []
        try:
            for line in open(self.path):
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        except OSError:
            pass
        finally:
            if self.path and os.path.exists(self.path):
                os.remove(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"], "samples": 0}
        def num(x):
            try:
                return float(x)
            except ValueError:
                return None
        sm = [num(r[1]) for r in rows if num(r[1]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i] == "Active"})
        # samples "under load": the SM clock above half of its maximum
        mx = num(rows[-1][2])
        loaded = [x for x in sm if mx is None or x > 0.5 * mx] or sm
        return {"sm_mhz": statistics.median(loaded) if loaded else None, "sm_max_mhz": mx,
                "reasons": reasons, "samples": len(rows),
                "power_w_max": max((num(r[3]) or 0.0) for r in rows)}


# ---------------------------------------------------------------------------------------
# workload
# ---------------------------------------------------------------------------------------

STACK_PREFIX = "stack_b"     # stack_b1, stack_b8, ...: the 32-layer decode stack
STACK_GRAPH = 8              # macro-steps per CUDA graph in the stack runs
EMBED_PREFIX = "embed_b"     # embed_b64, ...: the compositional embedder
EMBED_HANDLES = 8            # rotated handles: 8 x 32 MiB of weights > 129 MB L2
EMBED_TOK_PREFIX = "embedtok_b"  # embedtok_b64, ...: the embedder fed token ids
EMBED_TOK_HANDLES = 16       # rotated: 16 x 8 MiB of W_o > 129 MB L2 (and 3.7 GB of tables each)
FRONT_PREFIX = "qkv_front_b"  # qkv_front_b8, ...: the layer front (projection, RoPE, append)
FRONT_LAYERS = 8             # rotated layers: 8 x 48 MiB of fused weights > 129 MB L2
MICRO_PREFIX = "micro_b"     # micro_b8, ...: the micro-step decoder's attention


def workload(name):
    from paper_2505_20438_gb300 import workload as wl
    if name.startswith(STACK_PREFIX) and name[len(STACK_PREFIX):].isdigit():
        return wl.c4_sweep(int(name[len(STACK_PREFIX):]))
    if name.startswith(EMBED_PREFIX) and name[len(EMBED_PREFIX):].isdigit():
        return wl.embed_workload(int(name[len(EMBED_PREFIX):]))
    if name.startswith(EMBED_TOK_PREFIX) and name[len(EMBED_TOK_PREFIX):].isdigit():
        return wl.embed_tokens_workload(int(name[len(EMBED_TOK_PREFIX):]))
    if name.startswith(FRONT_PREFIX) and name[len(FRONT_PREFIX):].isdigit():
        return wl.front_workload(int(name[len(FRONT_PREFIX):]))
    if name.startswith(MICRO_PREFIX) and name[len(MICRO_PREFIX):].isdigit():
        return wl.micro_workload(int(name[len(MICRO_PREFIX):]))
    if name in wl.PREFILL_WORKLOADS:
        return wl.PREFILL_WORKLOADS[name]
    if name not in wl.WORKLOADS:
        raise SystemExit(f"unknown workload {name}; choose from "
                         f"{sorted(wl.WORKLOADS) + sorted(wl.PREFILL_WORKLOADS)} or "
                         f"{STACK_PREFIX}<batch>, {EMBED_PREFIX}<batch>, "
                         f"{EMBED_TOK_PREFIX}<batch>, {FRONT_PREFIX}<batch>, "
                         f"{MICRO_PREFIX}<batch>")
    return wl.WORKLOADS[name]


def base_counts(w):
    """Slots per sequence before the timed steps (uniform, or the workload's ragged draw)."""
    from paper_2505_20438_gb300 import workload as wl
    return wl.slot_counts(w, wl.rng_for(w.seed, 1))


STEP_TEXT = {
    "fused": "ham_decode_step: append of the slot (RoPE q,k) fused into attention over all slots",
    "split": "ham_kv_append (RoPE q,k + append) then ham_decode_attn over all slots",
}


def config_dict(w, path="fused", kv="bf16"):
    counts = base_counts(w)
    slots = w.slots if w.slot_range is None else (
        f"{int(counts.min())}..{int(counts.max())} (mean {counts.mean():.0f}, uniform draw "
        f"in [{w.slot_range[0]}, {w.slot_range[1]}])")
    return {"workload": w.name, "batch": w.batch, "n_q_heads": w.n_q_heads,
            "n_kv_heads": w.n_kv_heads, "head_dim": w.head_dim, "slots": slots,
            "page_slots": w.page_slots, "pages": "scattered by a seeded shuffle of a shared pool",
            "tokens_per_slot": "geometric p=0.5 capped at 4 (mean 1.875)",
            "step": STEP_TEXT[path],
            "kv_dtype": ("e4m3 codes + one int8 power-of-two exponent per (slot, KV head) row"
                         if kv == "fp8" else "bf16"),
            "l2": f"{CACHES} independent caches rotated ({CACHES} x "
                  f"{int(counts.sum()) * w.n_kv_heads * kv_row_bytes(w, kv) * 2 / 2**20:.0f} "
                  "MiB KV > 129 MB L2)",
            "graph": f"{GRAPH_STEPS} steps per CUDA graph, then each cache is rolled back "
                     "to its starting slot counts"}


def kv_row_bytes(w, kv="bf16"):
    """Bytes of one stored K (or V) row of one (slot, KV head): bf16 elements, or e4m3 codes
    plus the row's int8 exponent."""
    return w.head_dim + 1 if kv == "fp8" else w.head_dim * 2


def attn_bytes(w, lengths, kv="bf16"):
    """Algorithmic bytes of one attention launch over sequences of `lengths` slots: K and V
    of every slot once, q in, out, and the page-table entries."""
    kv = sum(int(L) for L in lengths) * w.n_kv_heads * kv_row_bytes(w, kv) * 2
    qo = 2 * w.batch * w.n_q_heads * w.head_dim * 2
    pt = sum(math.ceil(int(L) / w.page_slots) for L in lengths) * 4
    return kv + qo + pt


def append_bytes(w, kv="bf16"):
    """Algorithmic bytes of one append: q read+write, k_new/v_new in, K/V rows out, metadata."""
    return (2 * w.batch * w.n_q_heads * w.head_dim * 2 + 4 * w.batch * w.n_kv_heads * w.head_dim
            + 2 * w.batch * w.n_kv_heads * kv_row_bytes(w, kv) + w.batch * 4 * 6)


# ---------------------------------------------------------------------------------------
# our arm
# ---------------------------------------------------------------------------------------

def build_caches(w, device_index, rank, kv_dtype=0):
    import numpy as np
    import torch

    from paper_2505_20438_gb300 import ham
    from paper_2505_20438_gb300 import workload as wl

    caches = []
    counts_h = base_counts(w)
    lmax = int(counts_h.max())
    max_slots = lmax + GRAPH_STEPS // CACHES + 16
    for r in range(CACHES):
        seed = rank_cache_seed(w.seed, rank, r)
        kv = ham.ham_kv_alloc(1, w.batch, w.n_q_heads, w.n_kv_heads, w.head_dim, w.page_slots,
                              max_slots, pool_pages=int(math.ceil(
                                  w.batch * math.ceil(max_slots / w.page_slots) * w.pool_factor)),
                              page_seed=seed + 1, kv_dtype=kv_dtype)
        shape = (w.batch, lmax, w.n_kv_heads, w.head_dim)
        k = wl.device_normal_bf16(shape, w.value_scale, seed * 7 + 1)
        v = wl.device_normal_bf16(shape, w.value_scale, seed * 7 + 2)
        rng = wl.rng_for(seed, 5)
        ntok = wl.ntok_capped_geometric(rng, (w.batch, lmax))
        for b in range(w.batch):
            ntok[b, counts_h[b]:] = 0
        counts = torch.from_numpy(counts_h.astype(np.int32)).cuda()
        ham.ham_kv_fill(kv, 0, k, v, counts, ntok=torch.from_numpy(ntok).cuda())
        del k, v
        tokens = torch.from_numpy(ntok.sum(axis=1).astype(np.int64)).cuda()
        c = {
            "kv": kv, "counts": counts, "tokens": tokens,
            "q": wl.device_normal_bf16((w.batch, w.n_q_heads, w.head_dim), w.value_scale, seed * 7 + 3),
            "k_new": wl.device_normal_bf16((w.batch, w.n_kv_heads, w.head_dim), w.value_scale, seed * 7 + 4),
            "v_new": wl.device_normal_bf16((w.batch, w.n_kv_heads, w.head_dim), w.value_scale, seed * 7 + 5),
            "ntok_new": torch.from_numpy(wl.ntok_capped_geometric(rng, (w.batch,))).cuda(),
            "out": torch.empty((w.batch, w.n_q_heads, w.head_dim), dtype=torch.bfloat16, device="cuda"),
            "mean_ntok": float(ntok.sum() / max(1, counts_h.sum())),
        }
        caches.append(c)
    torch.cuda.synchronize()
    return caches


def run_ours(args, w):
    """The decode-step workload `w`; for the default Llama-8B layer (batch 8 x 4096 slots) the
    same line also carries the batch 8 x 8192 slots point (the target's "batch >= 8 and >= 8k
    slots"), measured the same way, under "target_point"."""
    import torch

    from paper_2505_20438_gb300 import build as build_mod
    from paper_2505_20438_gb300 import workload as wl

    rank, local_rank, world = dist_env()
    torch.cuda.set_device(local_rank)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    build_mod.build()
    result = measure_decode(args, w, rank, local_rank, world, args.min_seconds, full=True)
    if w.name == wl.C1_LLAMA8B.name and args.path == "fused" and not args.no_target_point:
        tp = measure_decode(args, wl.C1_LLAMA8B_S8K, rank, local_rank, world,
                            args.min_seconds / 2, full=False)
        result["target_point"] = {k: tp[k] for k in (
            "value", "unit", "steps", "ms_per_step", "kv_gbs", "kv_frac_of_measured_peak",
            "kv_frac_of_8tbs_spec", "slots_per_s", "tokens_per_s", "roofline", "gpu_launches",
            "clocks")}
        result["target_point"]["config"] = tp["config"]
        result["gpu_launches"] += tp["gpu_launches"]
    if rank == 0:
        print(json.dumps(result), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


def measure_decode(args, w, rank, local_rank, world, min_seconds, full):
    """Times the decode step of `w` over at least `min_seconds` (whole 64-step graphs); `full`
    adds the end-to-end arm and the CPU baseline.  Returns the bench line's fields."""
    import torch

    from paper_2505_20438_gb300 import ham

    fp8 = args.kv == "fp8"
    caches = build_caches(w, local_rank, rank, ham.HAM_KV_E4M3 if fp8 else ham.HAM_KV_BF16)
    stream = torch.cuda.Stream()
    n_graph = max(1, math.ceil(args.steps / GRAPH_STEPS))
    n_warm = max(1, math.ceil(max(args.warmup, 3) / GRAPH_STEPS))

    fused = args.path == "fused"

    def append_part(c):
        if not fused:
            ham.ham_kv_append(c["kv"], 0, c["q"], c["k_new"], c["v_new"], None, c["ntok_new"])

    def timed_part(c):
        if fused:
            ham.ham_decode_step(c["kv"], 0, c["q"], c["k_new"], c["v_new"], None, c["ntok_new"],
                                c["out"])
        else:
            ham.ham_decode_attn(c["kv"], 0, c["q"], c["out"])

    def one_step(c):
        append_part(c)
        timed_part(c)

    def rollback():
        for c in caches:
            ham.ham_kv_set_lengths(c["kv"], 0, c["counts"], c["tokens"])

    # eager warm-up (first launches configure the kernels outside of capture)
    with torch.cuda.stream(stream):
        for i in range(2 * CACHES):
            one_step(caches[i % CACHES])
        rollback()
    stream.synchronize()

    name = "ham_decode_step" if fused else "ham_decode_attn"
    try:
        span = (torch.cuda.Event(enable_timing=True, external=True),
                torch.cuda.Event(enable_timing=True, external=True))
        ev = [(torch.cuda.Event(enable_timing=True, external=True),
               torch.cuda.Event(enable_timing=True, external=True)) for _ in range(GRAPH_STEPS)]
        per_launch_method = (f"CUDA events before and after the {GRAPH_STEPS} consecutive {name} "
                             "calls of the last graph replay of the timed region (on the launching "
                             f"stream; programmatic dependent launch intact between them), / "
                             f"{GRAPH_STEPS}")
    except TypeError:
        span, ev = None, None
        per_launch_method = "timed region / steps (events inside graphs unavailable)"

    def capture(events):
        """events: None, "span" (around the steps, before the rollback) or "each" (around
        every step; that stops consecutive launches from overlapping)."""
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            if events == "span":
                span[0].record()
            for i in range(GRAPH_STEPS):
                c = caches[i % CACHES]
                append_part(c)
                if events == "each":
                    ev[i][0].record()
                timed_part(c)
                if events == "each":
                    ev[i][1].record()
            if events == "span":
                span[1].record()
            rollback()
        return g

    # the timed loop replays an event-free graph; the last replay is an identical graph with
    # events around its steps only (none between them)
    graph = capture(None)
    probe = capture("span") if span is not None else graph
    # fused: attention + combine/commit; split: append, attention, combine; then rollbacks
    launches_per_graph = (2 if fused else 3) * GRAPH_STEPS + CACHES

    # attended lengths inside one graph: step i (cache i % 4) sees counts + 1 + i // 4 slots
    counts_h = base_counts(w)
    attn_bytes_graph = sum(attn_bytes(w, counts_h + 1 + i // CACHES, args.kv)
                           for i in range(GRAPH_STEPS))
    step_bytes_graph = attn_bytes_graph + GRAPH_STEPS * append_bytes(w, args.kv)
    timed_bytes_graph = step_bytes_graph  # the span covers the whole step on both paths

    w0, w1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):          # replay() launches on the current stream
        for _ in range(n_warm):
            graph.replay()
        w0.record(stream)
        probe.replay()
        w1.record(stream)
    torch.cuda.synchronize()
    for c in caches:
        if ham.ham_kv_status(c["kv"]) != ham.HAM_DEVERR_NONE:
            raise RuntimeError("device error during warm-up")
    # whole graphs until the timed region lasts at least min_seconds, whatever --steps asks for
    graph_ms = max(w0.elapsed_time(w1), 1e-3)
    if world > 1:
        graph_ms = max_over_ranks(graph_ms, world, "cuda")
    n_graph = max(n_graph, min(100000, math.ceil(min_seconds * 1e3 / graph_ms)))
    steps = n_graph * GRAPH_STEPS

    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local_rank) as clocks, torch.cuda.stream(stream):
        t0.record(stream)
        for _ in range(n_graph - 1):
            graph.replay()
        probe.replay()
        t1.record(stream)
        torch.cuda.synchronize()
    elapsed_ms = max_over_ranks(t0.elapsed_time(t1), world, "cuda")
    if world > 1:
        torch.distributed.barrier()

    # the timed kernels' average duration in the loop (last replay of the timed region)
    if span is not None:
        attn_ms = [span[0].elapsed_time(span[1]) / GRAPH_STEPS] * GRAPH_STEPS
    else:
        attn_ms = [elapsed_ms / steps] * GRAPH_STEPS
    # and, after the timed region, the same launches one at a time (events around each)
    isolated_us = None
    if ev is not None:
        each = capture("each")
        with torch.cuda.stream(stream):
            each.replay()
        torch.cuda.synchronize()
        isolated_us = round(1e3 * statistics.mean(ev[i][0].elapsed_time(ev[i][1])
                                                  for i in range(GRAPH_STEPS)), 3)
    for c in caches:
        if ham.ham_kv_status(c["kv"]) != ham.HAM_DEVERR_NONE:
            raise RuntimeError("device error during the timed region")

    peak, peak_src = measured_peak_hbm()
    attn_gbs = timed_bytes_graph / (sum(attn_ms) * 1e-3) / 1e9
    ms_per_step = elapsed_ms / steps
    value = job_throughput(steps, world, elapsed_ms * 1e-3)
    step_gbs = world * n_graph * step_bytes_graph / (elapsed_ms * 1e-3) / 1e9
    mean_ntok = statistics.mean(c["mean_ntok"] for c in caches)

    e2e = run_e2e(args, w, caches, stream, rollback, world, one_step) if full else None

    traffic = profiled_traffic(("decode_step" if fused else "decode_attn") + ("_fp8" if fp8 else ""),
                               w.name, ATTN_FP8_SOURCES if fp8 else ATTN_SOURCES)
    result = {
        "metric": METRIC, "value": round(value, 2), "unit": UNIT, "n_gpus": world,
        "steps": steps, "steps_requested": args.steps, "timed_s": round(elapsed_ms * 1e-3, 3),
        "warmup": n_warm * GRAPH_STEPS, "ms_per_step": round(ms_per_step, 5),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "e4m3" if fp8 else "bf16",
        "accum_dtype": "f32", "data": "synthetic", "config": config_dict(w, args.path, args.kv),
        "kv_gbs": round(step_gbs, 1),
        "kv_frac_of_measured_peak": round(step_gbs / world / peak, 4),
        "kv_frac_of_8tbs_spec": round(step_gbs / world / 8000.0, 4),
        "slots_per_s": round(value * w.batch, 1),
        "tokens_per_s": round(value * w.batch * mean_ntok, 1),
        "roofline": {"bound": "hbm", "achieved": round(attn_gbs, 1), "peak": peak,
                     "unit": "GB/s", "frac": round(attn_gbs / peak, 4), "traffic": traffic,
                     "kernel": ((("decode_attn_fp8_kernel<bf16,step>" if fp8 else
                                  "decode_attn_kernel<128,bf16,step>") + " + combine_kernel<bf16,step>")
                                if fused else
                                ("append_kernel + " + ("decode_attn_fp8_kernel<bf16>" if fp8 else
                                 "decode_attn_kernel<128,bf16>") + " + combine_kernel<bf16>")),
                     "avg_launch_us": round(1e3 * statistics.mean(attn_ms), 3),
                     "isolated_launch_us": isolated_us,
                     "algorithmic_bytes_per_launch": int(timed_bytes_graph / GRAPH_STEPS),
                     "peak_source": peak_src, "duration_method": per_launch_method},
        "gpu_launches": n_graph * launches_per_graph * world,
        "e2e": e2e,
        "clocks": clocks.summary(),
        "cost_model": cost_model(mean_ntok, ms_per_step * 1e3),
    }
    if e2e is None:
        del result["e2e"]
    if fp8:
        result["mma_dtype"] = ("e4m3 codes read as stored by tcgen05 kind::f8f6f4 products (fp32 "
                               "accumulators in tensor memory); q 2^-f and the weights "
                               "p 2^(e_v - Gv + 7) as three e4m3 pieces each (~12 significant bits)")
    if full and rank == 0 and world == 1 and not args.no_cpu_baseline and not fp8:
        result["cpu_baseline"] = cpu_baseline(w, args.cpu_seconds)
    for c in caches:
        ham.ham_kv_free(c["kv"])
    return result


def cost_model(n, c_s_us, c_ratio=4.0 / 32.0):
    """Speed-up per macro-step of the paper's cost analysis (Sec. 3.7),
    r = n C(S) / (C(S) + (n - 1) c), as a MODELLED figure: n is the mean tokens per slot of the
    workload, C(S) this layer's measured decode step, and c (the micro-step decoder's cost per
    token) is assumed to be 4/32 of C(S), a 4-layer decoder against a 32-layer base model."""
    c = c_ratio * c_s_us
    return {"r": round(n * c_s_us / (c_s_us + (n - 1) * c), 4), "n": round(n, 4),
            "C_S_us": round(c_s_us, 3), "c_us": round(c, 3), "kind": "modelled",
            "assumption": "c = 4/32 of C(S): 4 micro-decoder layers against 32 base layers"}


def run_e2e(args, w, caches, stream, rollback, world, one_step):
    """Same steps through the public API with pinned host inputs copied in and the output
    copied back and read on the host every step.  Each cache's step (its host -> device input
    copies, the C-ABI call(s), the device -> host output copy) is captured once in a CUDA graph,
    as a serving loop would, so that the host issues one replay per step.  The caches are
    independent sequence sets, each on its own stream: a cache's steps stay in order on its
    stream, at most one step per cache is in flight, and before a cache's next step the host
    waits for its previous one and reads that step's output from pinned memory."""
    import numpy as np
    import torch
    from paper_2505_20438_gb300 import ham

    host = []
    for c in caches:
        host.append({k: c[k].cpu().pin_memory() for k in ("q", "k_new", "v_new", "ntok_new")})
        host[-1]["out"] = torch.empty(c["out"].shape, dtype=c["out"].dtype).pin_memory()
        host[-1]["out_bits"] = host[-1]["out"].view(torch.int16).numpy()  # the host's view
    h2d = sum(host[0][k].numel() * host[0][k].element_size() for k in ("q", "k_new", "v_new", "ntok_new"))
    d2h = host[0]["out"].numel() * host[0]["out"].element_size()
    n = max(GRAPH_STEPS, (args.e2e_steps // GRAPH_STEPS) * GRAPH_STEPS)
    per_cache = GRAPH_STEPS // CACHES  # steps of one cache between its rollbacks
    streams = [torch.cuda.Stream() for _ in caches]
    events = [torch.cuda.Event() for _ in caches]
    pending = [False] * len(caches)
    checksum = 0.0

    def io_step(j):
        c, h = caches[j], host[j]
        for k in ("q", "k_new", "v_new", "ntok_new"):
            c[k].copy_(h[k], non_blocking=True)
        one_step(c)
        h["out"].copy_(c["out"], non_blocking=True)

    with torch.cuda.stream(stream):
        for i in range(2 * CACHES):        # warm the eager path
            one_step(caches[i % CACHES])
        rollback()
    stream.synchronize()
    graphs = []
    for j, s_ in enumerate(streams):
        s_.wait_stream(stream)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s_):
            io_step(j)
        graphs.append(g)
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        rollback()                         # (capture issued no work; counts are as drawn)
    stream.synchronize()

    def settle(j):                # wait for cache j's step in flight and read its output
        nonlocal checksum
        if pending[j]:
            events[j].synchronize()
            bits = np.uint32(np.uint16(host[j]["out_bits"].flat[0])) << np.uint32(16)
            checksum += float(bits.view(np.float32))
            pending[j] = False

    if world > 1:
        torch.distributed.barrier()
    t = time.perf_counter()
    for i in range(n):
        j = i % CACHES
        settle(j)
        s_ = streams[j]
        with torch.cuda.stream(s_):
            graphs[j].replay()
            if (i // CACHES + 1) % per_cache == 0:      # this cache's rollback
                ham.ham_kv_set_lengths(caches[j]["kv"], 0, caches[j]["counts"], caches[j]["tokens"])
            events[j].record(s_)
        pending[j] = True
    for j in range(len(caches)):
        settle(j)
    dt = time.perf_counter() - t
    torch.cuda.synchronize()
    dt = max_over_ranks(dt, world, "cuda")
    return {"value": round(job_throughput(n, world, dt), 2), "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "steps": n,
            "path": f"every step: pinned host -> device copies of its inputs, the step's C-ABI "
                    f"call(s), device -> pinned host copy of its output (one CUDA graph per cache, "
                    f"replayed each step), the output read on the host; the {CACHES} independent "
                    f"caches each on their own stream, at most one step per cache in flight",
            "finite": math.isfinite(checksum)}


# ---------------------------------------------------------------------------------------
# CPU oracle: baseline leg and reference arm
# ---------------------------------------------------------------------------------------

def oracle_case(w):
    import oracle
    from paper_2505_20438_gb300 import workload as wl
    oracle.build()
    case = wl.make_case(w, extra_slots=4)
    return oracle, case, oracle.OracleCache.from_case(case)


def cpu_baseline(w, seconds):
    """Full macro-steps (append + attention of every head) of the oracle for ~`seconds`."""
    oracle, case, oc = oracle_case(w)
    n, t0 = 0, time.perf_counter()
    while True:
        q = case.q.copy()
        oc.append(case.k_new, case.v_new, case.ntok_new, q_inout=q)
        oc.decode_attn(q)
        oc.num_slots[:] = case.num_slots          # keep the workload at its slot count
        n += 1
        dt = time.perf_counter() - t0
        if dt >= seconds or n >= 10000:
            break
    # the same steps on one host thread, for a bounded few seconds
    n1, t1 = 0, time.perf_counter()
    while True:
        q = case.q.copy()
        oc.append(case.k_new, case.v_new, case.ntok_new, q_inout=q)
        oc.decode_attn(q, n_threads=1)
        oc.num_slots[:] = case.num_slots
        n1 += 1
        dt1 = time.perf_counter() - t1
        if dt1 >= min(3.0, seconds / 4) or n1 >= 1000:
            break
    return {"value": round(n / dt, 4), "unit": UNIT, "cores": oracle.max_threads(),
            "kind": "oracle", "single_thread_value": round(n1 / dt1, 4),
            "sample": f"{n} full macro-steps (append + attention of all {w.batch * w.n_q_heads} "
                      f"query heads over {w.slots} slots) of {w.name}, fp64 C oracle, "
                      f"OpenMP over (sequence, head); then {n1} on one thread"}


def run_reference_embed(args, w):
    """Reference arm of the embedder workload: the fp64 oracle, whole calls."""
    from oracle import embedder as oe
    from paper_2505_20438_gb300 import workload as wl
    c = embed_case(w)
    steps, warm = max(1, args.steps), max(3, args.warmup)
    # bounded: at most ~40 oracle calls in all
    steps, warm = min(steps, 30), min(warm, 10)
    for _ in range(warm):
        oe.embed(c.x, c.offsets, c.wq, c.wk, c.wv, c.wo, c.pos, w.n_heads)
    t0 = time.perf_counter()
    for _ in range(steps):
        oe.embed(c.x, c.offsets, c.wq, c.wk, c.wv, c.wo, c.pos, w.n_heads)
    value = steps / (time.perf_counter() - t0)
    unit = "calls/s"
    print(json.dumps({
        "impl": "reference",
        "metric": "compositional-embedder calls/s and achieved HBM GB/s (% of GB300 peak)",
        "value": round(value, 4), "unit": unit, "n_gpus": 1, "steps": steps, "warmup": warm,
        "ms_per_step": round(1e3 / value, 3), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.name, "batch": w.batch, "hidden": w.hidden,
                   "n_heads": w.n_heads},
        "cpu_baseline": {"value": round(value, 4), "unit": unit, "cores": os.cpu_count(),
                         "kind": "oracle",
                         "sample": f"{steps} whole calls of {w.name}" +
                                   (" (embeddings gathered from the table by the ids first)"
                                    if w.vocab else "")},
        "e2e": {"value": round(value, 4), "unit": unit, "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }), flush=True)


def run_reference(args, w):
    rank, _, world = dist_env()
    if rank != 0:
        return
    from paper_2505_20438_gb300 import workload as wl
    if isinstance(w, wl.EmbedWorkload):
        return run_reference_embed(args, w)
    if isinstance(w, wl.FrontWorkload):
        return run_reference_front(args, w)
    if isinstance(w, wl.MicroWorkload):
        return run_reference_micro(args, w)
    if isinstance(w, wl.PrefillWorkload):
        return run_reference_prefill(args, w)
    import dataclasses

    import oracle
    from paper_2505_20438_gb300 import workload as wl
    oracle.build()
    steps = max(1, args.steps)
    warm = max(3, args.warmup)
    # Each step runs the oracle as it stands (append + OpenMP attention of every head) on a
    # sub-case of the workload: fewer sequences, or one sequence with fewer slots, sized so
    # the whole run is about 40 full macro-steps of oracle work.  Attention work is linear
    # in the slot count, so the value is scaled by the sampled fraction of slots.
    total = int(base_counts(w).sum())          # slots attended by one layer's step
    mean_l = max(1, total // w.batch)
    frac = min(1.0, 40.0 / (steps + warm))
    if frac * w.batch >= 1.0:
        sub_b, sub_l = max(1, int(round(frac * w.batch))), mean_l
    else:
        sub_b, sub_l = 1, max(16, int(round(frac * total)))
    sub = dataclasses.replace(w, batch=sub_b, slots=sub_l, slot_range=None, layers=1)
    case = wl.make_case(sub, extra_slots=4)
    oc = oracle.OracleCache.from_case(case)
    def one():
        q = case.q.copy()
        oc.append(case.k_new, case.v_new, case.ntok_new, q_inout=q)
        oc.decode_attn(q)
        oc.num_slots[:] = case.num_slots
    for _ in range(warm):
        one()
    t0 = time.perf_counter()
    for _ in range(steps):
        one()
    dt = time.perf_counter() - t0
    share = (sub_b * sub_l) / total / w.layers  # a macro-step runs every layer
    value = steps * share / dt
    sample = (f"each step: append + attention of all heads for {sub_b} sequence(s) x {sub_l} "
              f"slots = {share:.4f} of a {w.name} macro-step; {steps} steps timed")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": UNIT,
        "n_gpus": world, "steps": steps, "warmup": warm,
        "ms_per_step": round(1e3 / value, 3), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic", "config": config_dict(w),
        "cpu_baseline": {"value": round(value, 4), "unit": UNIT, "cores": oracle.max_threads(),
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": round(value, 4), "unit": UNIT, "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }), flush=True)


def run_stack(args, w):
    """The decode stack: every macro-step runs ham_decode_step on each of the w.layers layers
    (one cache, one layer after the other, as a decoder does), STACK_GRAPH macro-steps per CUDA
    graph, then the layers are rolled back to their starting slot counts."""
    import numpy as np
    import torch

    from paper_2505_20438_gb300 import build as build_mod
    from paper_2505_20438_gb300 import ham
    from paper_2505_20438_gb300 import workload as wl

    rank, local_rank, world = dist_env()
    torch.cuda.set_device(local_rank)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    build_mod.build()
    B, L, layers = w.batch, w.slots, w.layers
    seed = rank_cache_seed(w.seed, rank, 0)
    max_slots = L + STACK_GRAPH + 16
    kv = ham.ham_kv_alloc(layers, B, w.n_q_heads, w.n_kv_heads, w.head_dim, w.page_slots,
                          max_slots, page_seed=seed + 1)
    rng = wl.rng_for(seed, 5)
    ntok_fill = wl.ntok_capped_geometric(rng, (B, L))
    counts = torch.full((B,), L, dtype=torch.int32, device="cuda")
    tokens = torch.from_numpy(ntok_fill.sum(axis=1).astype(np.int64)).cuda()
    ntok_fill_dev = torch.from_numpy(ntok_fill).cuda()
    for layer in range(layers):
        k = wl.device_normal_bf16((B, L, w.n_kv_heads, w.head_dim), w.value_scale,
                                  seed * 1000 + 10 * layer + 1)
        v = wl.device_normal_bf16((B, L, w.n_kv_heads, w.head_dim), w.value_scale,
                                  seed * 1000 + 10 * layer + 2)
        ham.ham_kv_fill(kv, layer, k, v, counts, ntok=ntok_fill_dev)
        del k, v
    shape_q, shape_kv = (B, w.n_q_heads, w.head_dim), (B, w.n_kv_heads, w.head_dim)
    q = [wl.device_normal_bf16(shape_q, w.value_scale, seed * 7 + 100 + l) for l in range(layers)]
    k_new = [wl.device_normal_bf16(shape_kv, w.value_scale, seed * 7 + 200 + l)
             for l in range(layers)]
    v_new = [wl.device_normal_bf16(shape_kv, w.value_scale, seed * 7 + 300 + l)
             for l in range(layers)]
    ntok_new = torch.from_numpy(wl.ntok_capped_geometric(rng, (B,))).cuda()
    out = [torch.empty(shape_q, dtype=torch.bfloat16, device="cuda") for _ in range(layers)]
    stream = torch.cuda.Stream()

    def macro_step():
        for l in range(layers):
            ham.ham_decode_step(kv, l, q[l], k_new[l], v_new[l], None, ntok_new, out[l])

    def rollback():
        for l in range(layers):
            ham.ham_kv_set_lengths(kv, l, counts, tokens)

    with torch.cuda.stream(stream):
        macro_step()
        rollback()
    stream.synchronize()
    span = (torch.cuda.Event(enable_timing=True, external=True),
            torch.cuda.Event(enable_timing=True, external=True))

    def capture(with_span):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            if with_span:
                span[0].record()
            for _ in range(STACK_GRAPH):
                macro_step()
            if with_span:
                span[1].record()
            rollback()
        return g

    graph, probe = capture(False), capture(True)
    # a macro-step runs every layer: at most 1024 of them keep the run within a minute or so
    n_graph = max(1, math.ceil(min(args.steps, 1024) / STACK_GRAPH))
    n_warm = max(1, math.ceil(max(args.warmup, 3) / STACK_GRAPH))
    steps = n_graph * STACK_GRAPH
    with torch.cuda.stream(stream):
        for _ in range(n_warm):
            graph.replay()
    torch.cuda.synchronize()
    if ham.ham_kv_status(kv) != ham.HAM_DEVERR_NONE:
        raise RuntimeError("device error during warm-up")
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local_rank) as clocks, torch.cuda.stream(stream):
        t0.record(stream)
        for _ in range(n_graph - 1):
            graph.replay()
        probe.replay()
        t1.record(stream)
        torch.cuda.synchronize()
    elapsed_ms = max_over_ranks(t0.elapsed_time(t1), world, "cuda")
    if world > 1:
        torch.distributed.barrier()
    if ham.ham_kv_status(kv) != ham.HAM_DEVERR_NONE:
        raise RuntimeError("device error during the timed region")
    counts_h = np.full(B, L)
    macro_bytes = layers * statistics.mean(attn_bytes(w, counts_h + 1 + m) + append_bytes(w)
                                           for m in range(STACK_GRAPH))
    span_us = 1e3 * span[0].elapsed_time(span[1]) / STACK_GRAPH
    peak, peak_src = measured_peak_hbm()
    value = job_throughput(steps, world, elapsed_ms * 1e-3)
    ms_per_step = elapsed_ms / steps
    achieved = macro_bytes / (span_us * 1e-6) / 1e9

    # end to end through the public API: every macro-step copies each layer's q, k_new, v_new
    # from pinned host memory, runs the stack and copies the last layer's output back, which the
    # host reads; the macro-step with its copies is captured once in a CUDA graph (as a serving
    # loop would: issued eagerly, the 96 copies and 32 calls of a macro-step are bound by the
    # host, not the GPU)
    host = {"q": [x.cpu().pin_memory() for x in q], "k": [x.cpu().pin_memory() for x in k_new],
            "v": [x.cpu().pin_memory() for x in v_new]}
    host_out = torch.empty(shape_q, dtype=torch.bfloat16).pin_memory()
    out_bits = host_out.view(torch.int16).numpy()
    h2d = layers * sum(x[0].numel() * x[0].element_size() for x in host.values())
    d2h = host_out.numel() * host_out.element_size()
    n_e2e = max(STACK_GRAPH, min(args.e2e_steps, 64) // STACK_GRAPH * STACK_GRAPH)
    io = torch.cuda.CUDAGraph()
    with torch.cuda.graph(io, stream=stream):
        for l in range(layers):
            q[l].copy_(host["q"][l], non_blocking=True)
            k_new[l].copy_(host["k"][l], non_blocking=True)
            v_new[l].copy_(host["v"][l], non_blocking=True)
        macro_step()
        host_out.copy_(out[-1], non_blocking=True)
    checksum = 0.0
    with torch.cuda.stream(stream):
        rollback()
        stream.synchronize()
        te = time.perf_counter()
        for i in range(n_e2e):
            io.replay()
            stream.synchronize()
            bits = np.uint32(np.uint16(out_bits.flat[0])) << np.uint32(16)
            checksum += float(bits.view(np.float32))      # the host reads the step's result
            if (i + 1) % STACK_GRAPH == 0:
                rollback()
        stream.synchronize()
        dte = time.perf_counter() - te
    dte = max_over_ranks(dte, world, "cuda")

    mean_ntok = float(ntok_fill.mean())
    result = {
        "metric": METRIC, "value": round(value, 2), "unit": UNIT, "n_gpus": world,
        "steps": steps, "warmup": n_warm * STACK_GRAPH, "ms_per_step": round(ms_per_step, 5),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "accum_dtype": "f32", "data": "synthetic",
        "config": {"workload": w.name, "layers": layers, "batch": B, "n_q_heads": w.n_q_heads,
                   "n_kv_heads": w.n_kv_heads, "head_dim": w.head_dim,
                   "slots": f"{L} at the start of each graph, +1 per macro-step",
                   "page_slots": w.page_slots,
                   "pages": "scattered by a seeded shuffle of the pool",
                   "tokens_per_slot": "geometric p=0.5 capped at 4",
                   "step": f"one macro-step: ham_decode_step on each of the {layers} layers",
                   "l2": f"{layers} layers of KV ({layers * B * L * w.n_kv_heads * w.head_dim * 4 / 2**20:.0f} MiB) > 129 MB L2",
                   "graph": f"{STACK_GRAPH} macro-steps per CUDA graph, then every layer is "
                            "rolled back"},
        "kv_gbs": round(macro_bytes * value / 1e9, 1),
        "kv_frac_of_measured_peak": round(macro_bytes * value / world / 1e9 / peak, 4),
        "slots_per_s": round(value * B, 1),
        "tokens_per_s": round(value * B * mean_ntok, 1),
        "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                     "frac": round(achieved / peak, 4), "traffic": None,
                     "kernel": "decode_attn_kernel<128,bf16,step> + combine_kernel<bf16,step>, "
                               f"{layers} layers",
                     "avg_launch_us": round(span_us / layers, 3),
                     "algorithmic_bytes_per_launch": int(macro_bytes / layers),
                     "peak_source": peak_src,
                     "duration_method": f"CUDA events around the {STACK_GRAPH} macro-steps of the "
                                        f"last graph replay, / ({STACK_GRAPH} x {layers})"},
        "gpu_launches": n_graph * (STACK_GRAPH * layers * 2 + layers) * world,
        "e2e": {"value": round(job_throughput(n_e2e, world, dte), 2), "unit": UNIT,
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": n_e2e,
                "finite": math.isfinite(checksum),
                "path": "every macro-step: pinned host -> device copies of every layer's q, k_new, "
                        "v_new, the 32 layers' ham_decode_step, device -> pinned host copy of the "
                        "last layer's output, read on the host (one CUDA graph, replayed)"},
        "clocks": clocks.summary(),
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import dataclasses
        one = cpu_baseline(dataclasses.replace(w, layers=1), args.cpu_seconds)
        one["value"] = round(one["value"] / layers, 4)
        one["single_thread_value"] = round(one["single_thread_value"] / layers, 4)
        one["sample"] += f"; one layer's steps, divided by {layers} layers"
        result["cpu_baseline"] = one
    if rank == 0:
        print(json.dumps(result), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


def embed_case(w):
    """The seeded case of an embedder workload; for token ids, case.x = table[ids]."""
    from paper_2505_20438_gb300 import workload as wl
    return wl.make_embed_tokens_case(w, w.vocab).case if w.vocab else wl.make_embed_case(w)


def embed_bytes(w, T, B, singles=0):
    """Algorithmic bytes of one call.  Embeddings given: the four H x H bf16 weights and the
    fp32 position terms once, the token embeddings and offsets in, the fused states out.
    Token ids: W_o and the position terms once, the tabulated fp32 projections of each token
    (12 H bytes), the embedding rows of the single-token sequences, the ids and offsets in,
    the states out."""
    H = w.hidden
    io = w.max_patch * 2 * H * 4 + (B + 1) * 4 + B * H * 2
    if w.vocab:
        return H * H * 2 + io + T * 3 * H * 4 + singles * H * 2 + T * 4
    return 4 * H * H * 2 + io + T * H * 2


def run_embed(args, w):
    """The compositional embedder: one call fuses the last macro-step's tokens of w.batch
    sequences, given as embeddings or (w.vocab > 0) as token ids; calls rotate over handles
    whose weights together far exceed L2, 64 calls per CUDA graph."""
    import numpy as np
    import torch

    from paper_2505_20438_gb300 import build as build_mod
    from paper_2505_20438_gb300 import ham
    from paper_2505_20438_gb300 import workload as wl

    rank, local_rank, world = dist_env()
    torch.cuda.set_device(local_rank)
    if world > 1 and not torch.distributed.is_initialized():
        torch.distributed.init_process_group("nccl")
    build_mod.build()
    tc = wl.make_embed_tokens_case(w, w.vocab) if w.vocab else None
    c = tc.case if tc else wl.make_embed_case(w)
    B, H, T = w.batch, w.hidden, int(c.offsets[-1])
    n_handles = EMBED_TOK_HANDLES if w.vocab else EMBED_HANDLES

    def dev(bits):
        return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()

    weights = [dev(a) for a in (c.wq, c.wk, c.wv, c.wo)]
    pos = dev(c.pos)
    handles = [ham.ham_embedder_alloc(H, w.n_heads, B, w.max_patch, *weights, pos)
               for _ in range(n_handles)]
    del weights
    x = dev(c.x)
    offsets = torch.from_numpy(c.offsets).cuda()
    ids = None
    if tc:
        table = dev(tc.table)
        for e in handles:
            ham.ham_embedder_set_vocab(e, table)
        del table
        ids = torch.from_numpy(tc.ids).cuda()

    def call(e, out):
        if ids is not None:
            ham.ham_embed_tokens(e, ids, offsets, out)
        else:
            ham.ham_embed(e, x, offsets, out)
    outs = [torch.empty((B, H), dtype=torch.bfloat16, device="cuda") for _ in handles]
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        for j, e in enumerate(handles):        # eager first calls
            call(e, outs[j])
    stream.synchronize()
    span = (torch.cuda.Event(enable_timing=True, external=True),
            torch.cuda.Event(enable_timing=True, external=True))

    def capture(with_span):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            if with_span:
                span[0].record()
            for i in range(GRAPH_STEPS):
                j = i % n_handles
                call(handles[j], outs[j])
            if with_span:
                span[1].record()
        return g

    graph, probe = capture(False), capture(True)
    n_graph = max(1, math.ceil(min(args.steps, 8192) / GRAPH_STEPS))
    n_warm = max(1, math.ceil(max(args.warmup, 3) / GRAPH_STEPS))
    steps = n_graph * GRAPH_STEPS
    with torch.cuda.stream(stream):
        for _ in range(n_warm):
            graph.replay()
    torch.cuda.synchronize()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local_rank) as clocks, torch.cuda.stream(stream):
        t0.record(stream)
        for _ in range(n_graph - 1):
            graph.replay()
        probe.replay()
        t1.record(stream)
        torch.cuda.synchronize()
    elapsed_ms = max_over_ranks(t0.elapsed_time(t1), world, "cuda")
    if world > 1:
        torch.distributed.barrier()
    for e in handles:
        if ham.ham_embedder_status(e) != ham.HAM_DEVERR_NONE:
            raise RuntimeError("device error during the timed region")
    call_us = 1e3 * span[0].elapsed_time(span[1]) / GRAPH_STEPS
    nbytes = embed_bytes(w, T, B, singles=int((c.counts == 1).sum()))
    peak, peak_src = measured_peak_hbm()
    value = job_throughput(steps, world, elapsed_ms * 1e-3)
    achieved = nbytes / (call_us * 1e-6) / 1e9

    # end to end: each call copies the tokens and offsets from pinned host memory, fuses them
    # and copies the states back; one graph per handle, the host reads every call's result
    src = ids if ids is not None else x   # the call's token input: ids or embeddings
    hx, hoff = src.cpu().pin_memory(), offsets.cpu().pin_memory()
    hout = torch.empty((B, H), dtype=torch.bfloat16).pin_memory()
    hbits = hout.view(torch.int16).numpy()
    io = []
    for j, e in enumerate(handles):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            src.copy_(hx, non_blocking=True)
            offsets.copy_(hoff, non_blocking=True)
            call(e, outs[j])
            hout.copy_(outs[j], non_blocking=True)
        io.append(g)
    torch.cuda.synchronize()
    n_e2e = max(GRAPH_STEPS, (args.e2e_steps // GRAPH_STEPS) * GRAPH_STEPS)
    checksum = 0.0
    te = time.perf_counter()
    with torch.cuda.stream(stream):
        for i in range(n_e2e):
            io[i % n_handles].replay()
            stream.synchronize()
            bits = np.uint32(np.uint16(hbits.flat[0])) << np.uint32(16)
            checksum += float(bits.view(np.float32))
    dte = max_over_ranks(time.perf_counter() - te, world, "cuda")

    result = {
        "metric": "compositional-embedder calls/s and achieved HBM GB/s (% of GB300 peak)",
        "value": round(value, 2), "unit": "calls/s", "n_gpus": world, "steps": steps,
        "warmup": n_warm * GRAPH_STEPS, "ms_per_step": round(elapsed_ms / steps, 5),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "accum_dtype": "f32", "data": "synthetic",
        "config": {"workload": w.name, "batch": B, "hidden": H, "n_heads": w.n_heads,
                   "tokens": T, "fused_sequences": int((c.counts > 1).sum()),
                   "tokens_per_sequence": "geometric p=0.5 capped at 4",
                   "vocab": w.vocab or None,
                   "step": ("one ham_embed_tokens call: gather of the tabulated projections "
                            "with fusion, output GEMM, finish" if w.vocab else
                            "one ham_embed call: QKV GEMM, fusion, output GEMM, finish"),
                   "l2": f"{n_handles} handles rotated ({n_handles} x "
                         f"{(1 if w.vocab else 4) * H * H * 2 / 1e6:.1f} MB of weights "
                         f"> 129 MB L2)",
                   "graph": f"{GRAPH_STEPS} calls per CUDA graph"},
        "sequences_per_s": round(value * B, 1),
        "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                     "frac": round(achieved / peak, 4), "traffic": None,
                     "kernel": ("fuse_kernel (gather) + gemm_xwt_kernel (output projection) "
                                "+ finish_kernel" if w.vocab else
                                "gemm_xwt_kernel (Q/K/V projection) + fuse_kernel + "
                                "gemm_xwt_kernel (output projection) + finish_kernel"),
                     "avg_launch_us": round(call_us, 3),
                     "algorithmic_bytes_per_launch": int(nbytes),
                     "peak_source": peak_src,
                     "duration_method": f"CUDA events around the {GRAPH_STEPS} calls of the "
                                        "last graph replay, / " + str(GRAPH_STEPS)},
        "gpu_launches": n_graph * GRAPH_STEPS * 2 * world,
        "e2e": {"value": round(job_throughput(n_e2e, world, dte), 2), "unit": "calls/s",
                "h2d_bytes_per_step": src.numel() * src.element_size() + (B + 1) * 4,
                "d2h_bytes_per_step": B * H * 2,
                "steps": n_e2e, "finite": math.isfinite(checksum),
                "path": "every call: pinned host -> device copies of the tokens "
                        f"({'ids' if w.vocab else 'embeddings'}) and offsets, the call, device "
                        "-> pinned host copy of the states, read on the host (one CUDA graph "
                        "per handle)"},
        "clocks": clocks.summary(),
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        result["cpu_baseline"] = embed_cpu_baseline(c, args.cpu_seconds)
    for e in handles:
        ham.ham_embedder_free(e)
    if rank == 0:
        print(json.dumps(result), flush=True)


def embed_cpu_baseline(c, seconds):
    """The fp64 oracle on the host cores (numpy), whole calls for about `seconds`."""
    from oracle import embedder as oe
    n, t0 = 0, time.perf_counter()
    while True:
        oe.embed(c.x, c.offsets, c.wq, c.wk, c.wv, c.wo, c.pos, c.w.n_heads)
        n += 1
        dt = time.perf_counter() - t0
        if dt >= seconds or n >= 1000:
            break
    return {"value": round(n / dt, 4), "unit": "calls/s", "cores": os.cpu_count(),
            "kind": "oracle",
            "sample": f"{n} whole calls of {c.w.name} (fp64 numpy oracle; its matrix products "
                      f"may use every core)"}


# ---------------------------------------------------------------------------------------
# macro-step layer front (q/k/v projection, RoPE, append)
# ---------------------------------------------------------------------------------------

FRONT_METRIC = "layer-front calls/s (q/k/v projection + RoPE + append) and achieved HBM GB/s"


def front_bytes(w, kv="bf16"):
    """Algorithmic bytes of one call: the fused weight once, x in, q_rot out, the new K and V
    rows (FP8 pools: codes and one exponent byte a row), and per sequence its counters, token
    count, page-table entry and slot metadata (4 + 4 + 8 + 4 read, 4 + 4 + 4 + 8 written)."""
    B, H, d = w.batch, w.hidden, w.head_dim
    row = d + 1 if kv == "fp8" else d * 2
    return (w.out_rows * H * 2 + B * H * 2 + B * w.n_q_heads * d * 2 +
            B * 2 * w.n_kv_heads * row + B * 40)


def front_cpu_sample(w, seconds, max_calls=1000):
    """The fp64 oracle front (numpy) on whole calls for about `seconds`; returns (calls, s)."""
    import dataclasses

    import numpy as np

    import oracle
    from oracle import front as ofront
    from paper_2505_20438_gb300 import workload as wl
    oracle.build()
    cw = wl.Workload("front_cache", batch=w.batch, n_q_heads=w.n_q_heads,
                     n_kv_heads=w.n_kv_heads, head_dim=w.head_dim, page_slots=16, layers=1,
                     seed=w.seed)
    case = wl.make_case(cw, num_slots=np.zeros(w.batch, np.int32), extra_slots=16)
    oc = oracle.OracleCache.from_case(case)
    x, W = wl.front_inputs(w)
    ntok = np.ones(w.batch, np.int32)
    n, t0 = 0, time.perf_counter()
    while True:
        ofront.qkv_append(oc, x, W, ntok)
        oc.num_slots[:] = 0
        n += 1
        dt = time.perf_counter() - t0
        if dt >= seconds or n >= max_calls:
            return n, dt


def run_reference_front(args, w):
    """Reference arm of the layer front: the fp64 oracle, whole calls (bounded)."""
    steps, warm = min(max(1, args.steps), 30), min(max(3, args.warmup), 5)
    warm, _ = front_cpu_sample(w, 1e9, max_calls=warm)
    n, dt = front_cpu_sample(w, 1e9, max_calls=steps)
    value = n / dt
    print(json.dumps({
        "impl": "reference", "metric": FRONT_METRIC, "value": round(value, 4),
        "unit": "calls/s", "n_gpus": 1, "steps": n, "warmup": warm,
        "ms_per_step": round(1e3 / value, 3), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.name, "batch": w.batch, "hidden": w.hidden,
                   "n_q_heads": w.n_q_heads, "n_kv_heads": w.n_kv_heads,
                   "head_dim": w.head_dim},
        "cpu_baseline": {"value": round(value, 4), "unit": "calls/s", "cores": os.cpu_count(),
                         "kind": "oracle", "sample": f"{n} whole calls of {w.name}"},
        "e2e": {"value": round(value, 4), "unit": "calls/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }), flush=True)


def run_front(args, w):
    """The layer front: one call projects x of w.batch sequences with one layer's fused
    weight, rotates q and k at the new slot's position and appends the slot.  Calls rotate
    over FRONT_LAYERS layers of one cache, each with its own weight (together far above L2),
    64 calls per CUDA graph; each graph ends by rolling every layer back to its starting
    length.  cuBLAS's GEMM of the same projection (no RoPE, no append) is timed the same way
    for context."""
    import numpy as np
    import torch

    from paper_2505_20438_gb300 import build as build_mod
    from paper_2505_20438_gb300 import ham
    from paper_2505_20438_gb300 import workload as wl

    rank, local_rank, world = dist_env()
    torch.cuda.set_device(local_rank)
    if world > 1 and not torch.distributed.is_initialized():
        torch.distributed.init_process_group("nccl")
    build_mod.build()
    B, H, L = w.batch, w.hidden, FRONT_LAYERS
    per_layer = GRAPH_STEPS // L
    start = 256                                   # slots per sequence before every graph
    fp8 = args.kv == "fp8"
    kv = ham.ham_kv_alloc(L, B, w.n_q_heads, w.n_kv_heads, w.head_dim, 16,
                          start + per_layer + 8, page_seed=1 + rank,
                          kv_dtype=ham.HAM_KV_E4M3 if fp8 else ham.HAM_KV_BF16)
    lengths = torch.full((B,), start, dtype=torch.int32, device="cuda")
    tokens = torch.full((B,), 2 * start, dtype=torch.int64, device="cuda")
    for layer in range(L):
        ham.ham_kv_set_lengths(kv, layer, lengths, tokens)
    weights = [wl.device_normal_bf16((w.out_rows, H), 1.0 / math.sqrt(H), 1000 * w.seed + 10 * rank + j)
               for j in range(L)]
    x = wl.device_normal_bf16((B, H), 1.0, 1000 * w.seed + 10 * rank + 99)
    ntok = torch.from_numpy(wl.ntok_capped_geometric(wl.rng_for(w.seed + rank, 9), (B,))).cuda()
    q_rot = torch.empty((B, w.n_q_heads, w.head_dim), dtype=torch.bfloat16, device="cuda")
    y = torch.empty((B, w.out_rows), dtype=torch.bfloat16, device="cuda")
    stream = torch.cuda.Stream()
    span = (torch.cuda.Event(enable_timing=True, external=True),
            torch.cuda.Event(enable_timing=True, external=True))

    def capture(fn, with_span):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            if with_span:
                span[0].record()
            for i in range(GRAPH_STEPS):
                fn(i % L)
            if with_span:
                span[1].record()
            for layer in range(L):
                ham.ham_kv_set_lengths(kv, layer, lengths, tokens)
        return g

    def call(layer):
        ham.ham_qkv_append(kv, layer, x, weights[layer], ntok, q_rot)

    def gemm(layer):
        torch.matmul(x, weights[layer].t(), out=y)

    with torch.cuda.stream(stream):
        for layer in range(L):                       # eager first calls
            call(layer)
            gemm(layer)
        for layer in range(L):
            ham.ham_kv_set_lengths(kv, layer, lengths, tokens)
    stream.synchronize()
    graph, probe = capture(call, False), capture(call, True)
    n_graph = max(1, math.ceil(min(args.steps, 16384) / GRAPH_STEPS))
    n_warm = max(1, math.ceil(max(args.warmup, 3) / GRAPH_STEPS))
    steps = n_graph * GRAPH_STEPS
    with torch.cuda.stream(stream):
        for _ in range(n_warm):
            graph.replay()
    torch.cuda.synchronize()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local_rank) as clocks, torch.cuda.stream(stream):
        t0.record(stream)
        for _ in range(n_graph - 1):
            graph.replay()
        probe.replay()
        t1.record(stream)
        torch.cuda.synchronize()
    elapsed_ms = max_over_ranks(t0.elapsed_time(t1), world, "cuda")
    if world > 1:
        torch.distributed.barrier()
    call_us = 1e3 * span[0].elapsed_time(span[1]) / GRAPH_STEPS
    if ham.ham_kv_status(kv) != ham.HAM_DEVERR_NONE:
        raise RuntimeError("device error during the timed region")
    # cuBLAS's GEMM of the same projection, timed the same way (context only)
    gprobe = capture(gemm, True)
    with torch.cuda.stream(stream):
        for _ in range(3):
            gprobe.replay()
    torch.cuda.synchronize()
    gemm_us = 1e3 * span[0].elapsed_time(span[1]) / GRAPH_STEPS

    nbytes = front_bytes(w, args.kv)
    peak, peak_src = measured_peak_hbm()
    value = job_throughput(steps, world, elapsed_ms * 1e-3)
    achieved = nbytes / (call_us * 1e-6) / 1e9

    # end to end: each call copies x and ntok from pinned host memory, runs the front and
    # copies q_rot back; one graph per layer, the host reads every call's result
    hx, hn = x.cpu().pin_memory(), ntok.cpu().pin_memory()
    hq = torch.empty_like(q_rot, device="cpu").pin_memory()
    hbits = hq.view(torch.int16).numpy()
    io = []
    for layer in range(L):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            x.copy_(hx, non_blocking=True)
            ntok.copy_(hn, non_blocking=True)
            call(layer)
            ham.ham_kv_set_lengths(kv, layer, lengths, tokens)
            hq.copy_(q_rot, non_blocking=True)
        io.append(g)
    torch.cuda.synchronize()
    n_e2e = max(GRAPH_STEPS, (args.e2e_steps // GRAPH_STEPS) * GRAPH_STEPS)
    checksum = 0.0
    te = time.perf_counter()
    with torch.cuda.stream(stream):
        for i in range(n_e2e):
            io[i % L].replay()
            stream.synchronize()
            bits = np.uint32(np.uint16(hbits.flat[0])) << np.uint32(16)
            checksum += float(bits.view(np.float32))
    dte = max_over_ranks(time.perf_counter() - te, world, "cuda")
    if ham.ham_kv_status(kv) != ham.HAM_DEVERR_NONE:
        raise RuntimeError("device error in the end-to-end loop")

    result = {
        "metric": FRONT_METRIC, "value": round(value, 2), "unit": "calls/s", "n_gpus": world,
        "steps": steps, "warmup": n_warm * GRAPH_STEPS,
        "ms_per_step": round(elapsed_ms / steps, 5), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "accum_dtype": "f32",
        "data": "synthetic",
        "config": {"workload": w.name, "batch": B, "hidden": H, "n_q_heads": w.n_q_heads,
                   "n_kv_heads": w.n_kv_heads, "head_dim": w.head_dim,
                   "weights": "fused [W_q; W_k; W_v] bf16 N(0, 1/H), x N(0, 1)",
                   "step": "one ham_qkv_append call: projection, RoPE of q and k, append",
                   "kv_dtype": ("e4m3 codes + one int8 power-of-two exponent per row (encoded "
                                "by the front)" if fp8 else "bf16"),
                   "l2": f"{L} layers' weights rotated ({L} x {w.out_rows * H * 2 / 2**20:.0f} "
                         f"MiB > 129 MB L2)",
                   "graph": f"{GRAPH_STEPS} calls per CUDA graph, then {L} counter rollbacks"},
        "sequences_per_s": round(value * B, 1),
        "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                     "frac": round(achieved / peak, 4),
                     "traffic": None if fp8 else profiled_traffic("front", w.name, FRONT_SOURCES),
                     "kernel": "front_kernel", "avg_launch_us": round(call_us, 3),
                     "algorithmic_bytes_per_launch": int(nbytes), "peak_source": peak_src,
                     "duration_method": f"CUDA events around the {GRAPH_STEPS} calls of the "
                                        f"last graph replay, / {GRAPH_STEPS}"},
        "cublas_gemm_same_projection_us": round(gemm_us, 3),
        "gpu_launches": n_graph * (GRAPH_STEPS + L) * world,
        "e2e": {"value": round(job_throughput(n_e2e, world, dte), 2), "unit": "calls/s",
                "h2d_bytes_per_step": B * H * 2 + B * 4,
                "d2h_bytes_per_step": B * w.n_q_heads * w.head_dim * 2,
                "steps": n_e2e, "finite": math.isfinite(checksum),
                "path": "every call: pinned host -> device copies of x and ntok, the call, a "
                        "counter rollback, device -> pinned host copy of q_rot, read on the "
                        "host (one CUDA graph per layer)"},
        "clocks": clocks.summary(),
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        n, dt = front_cpu_sample(w, args.cpu_seconds)
        result["cpu_baseline"] = {"value": round(n / dt, 4), "unit": "calls/s",
                                  "cores": os.cpu_count(), "kind": "oracle",
                                  "sample": f"{n} whole calls of {w.name} (fp64 numpy oracle; "
                                            f"its matrix product may use every core)"}
    ham.ham_kv_free(kv)
    if rank == 0:
        print(json.dumps(result), flush=True)


# ---------------------------------------------------------------------------------------
# micro-step decoder attention (local cache of the context entries and the micro-tokens)
# ---------------------------------------------------------------------------------------

MICRO_METRIC = "micro-steps/s of the micro-step decoder's attention (all its layers, one launch each)"


def micro_call_bytes(w, old):
    """Algorithmic bytes of one ham_micro_step call when every sequence holds `old` slots: the old
    K/V rows, q, k_new, v_new in, out, the new K/V rows out, per sequence its counters, token
    count, page-table entry and slot metadata (20 B read, 20 B written)."""
    B, Hq, Hkv, d = w.batch, w.n_q_heads, w.n_kv_heads, w.head_dim
    return (B * old * Hkv * d * 4 + B * Hq * d * 2 * 2 + B * Hkv * d * 4 * 2 + B * 40)


def micro_cpu_sample(w, seconds, max_steps=100000):
    """The fp64 oracle on whole micro-steps (append + attention of every layer) of the workload;
    returns (micro-steps, seconds)."""
    import numpy as np

    import oracle
    from paper_2505_20438_gb300 import workload as wl
    oracle.build()
    case = wl.make_micro_case(w)
    caches = [oracle.OracleCache.from_case(case) for _ in range(w.layers)]
    n, t0 = 0, time.perf_counter()
    while True:
        for i in range(w.micro_steps):
            for oc in caches:
                q = case.q.copy()
                oc.append(case.k_new, case.v_new, case.ntok_new, q_inout=q)
                oc.decode_attn(q, n_threads=1)
            n += 1
        for oc in caches:
            oc.num_slots[:] = case.num_slots
        dt = time.perf_counter() - t0
        if dt >= seconds or n >= max_steps:
            return n, dt


def run_reference_micro(args, w):
    """Reference arm of the micro-step workload: the fp64 oracle, whole micro-steps (bounded)."""
    steps, warm = min(max(1, args.steps), 3000), min(max(3, args.warmup), 30)
    warm, _ = micro_cpu_sample(w, 1e9, max_steps=warm)
    n, dt = micro_cpu_sample(w, 1e9, max_steps=steps)
    value = n / dt
    print(json.dumps({
        "impl": "reference", "metric": MICRO_METRIC, "value": round(value, 4),
        "unit": "micro-steps/s", "n_gpus": 1, "steps": n, "warmup": warm,
        "ms_per_step": round(1e3 / value, 4), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.name, "batch": w.batch, "layers": w.layers,
                   "context": w.context, "micro_steps": w.micro_steps},
        "cpu_baseline": {"value": round(value, 4), "unit": "micro-steps/s", "cores": 1,
                         "kind": "oracle", "sample": f"{n} micro-steps of {w.name}"},
        "e2e": {"value": round(value, 4), "unit": "micro-steps/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }), flush=True)


def run_micro(args, w):
    """The micro-step decoder's attention: each macro-step, every sequence's local cache holds
    w.context entries (hidden states of middle layers of the base model); the decoder then runs
    w.micro_steps micro-steps, each a ham_micro_step call on every one of its w.layers layers
    (append the micro-token's key and value, attend over the local entries), and the local
    cache is rolled back to the context for the next macro-step.  16 macro-steps per CUDA graph;
    ham_decode_step on the same handle is timed the same way for context."""
    import numpy as np
    import torch

    from paper_2505_20438_gb300 import build as build_mod
    from paper_2505_20438_gb300 import ham
    from paper_2505_20438_gb300 import workload as wl

    rank, local_rank, world = dist_env()
    torch.cuda.set_device(local_rank)
    if world > 1 and not torch.distributed.is_initialized():
        torch.distributed.init_process_group("nccl")
    build_mod.build()
    B, L, C, M = w.batch, w.layers, w.context, w.micro_steps
    case = wl.make_micro_case(dataclasses_replace_seed(w, rank))
    kv = ham.ham_kv_alloc(L, B, w.n_q_heads, w.n_kv_heads, w.head_dim, 16, C + M + 1,
                          page_seed=1 + rank)

    def dev(bits):
        return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()

    k_ctx, v_ctx = dev(case.k), dev(case.v)
    counts = torch.from_numpy(case.num_slots).cuda()
    tokens = torch.full((B,), C, dtype=torch.int64, device="cuda")
    for layer in range(L):
        ham.ham_kv_fill(kv, layer, k_ctx, v_ctx, counts)
    # per (micro-step, layer) inputs: distinct draws, resident on the device
    rng = wl.rng_for(w.seed + rank, 31)
    qs = [[dev(wl.normal_bf16(rng, (B, w.n_q_heads, w.head_dim))) for _ in range(L)] for _ in range(M)]
    ks = [[dev(wl.normal_bf16(rng, (B, w.n_kv_heads, w.head_dim))) for _ in range(L)] for _ in range(M)]
    vs = [[dev(wl.normal_bf16(rng, (B, w.n_kv_heads, w.head_dim))) for _ in range(L)] for _ in range(M)]
    ntok = torch.ones(B, dtype=torch.int32, device="cuda")
    outs = [torch.empty((B, w.n_q_heads, w.head_dim), dtype=torch.bfloat16, device="cuda")
            for _ in range(L)]
    stream = torch.cuda.Stream()
    span = (torch.cuda.Event(enable_timing=True, external=True),
            torch.cuda.Event(enable_timing=True, external=True))
    MACRO = 16

    def macro_step(fn, with_span=False):
        for i in range(M):
            if with_span and i == 0:
                span[0].record()
            for layer in range(L):
                fn(kv, layer, qs[i][layer], ks[i][layer], vs[i][layer], None, ntok, outs[layer])
            if with_span and i == M - 1:
                span[1].record()
        for layer in range(L):
            ham.ham_kv_set_lengths(kv, layer, counts, tokens)

    def capture(fn, with_span):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for r in range(MACRO):
                macro_step(fn, with_span and r == MACRO - 1)
        return g

    with torch.cuda.stream(stream):
        macro_step(ham.ham_micro_step)
        macro_step(ham.ham_decode_step)
    stream.synchronize()
    graph, probe = capture(ham.ham_micro_step, False), capture(ham.ham_micro_step, True)
    n_graph = max(1, math.ceil(min(args.steps, 40960) / (MACRO * M)))
    n_warm = max(1, math.ceil(max(args.warmup, 3) / (MACRO * M)))
    steps = n_graph * MACRO * M
    with torch.cuda.stream(stream):
        for _ in range(n_warm):
            graph.replay()
    torch.cuda.synchronize()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local_rank) as clocks, torch.cuda.stream(stream):
        t0.record(stream)
        for _ in range(n_graph - 1):
            graph.replay()
        probe.replay()
        t1.record(stream)
        torch.cuda.synchronize()
    elapsed_ms = max_over_ranks(t0.elapsed_time(t1), world, "cuda")
    if world > 1:
        torch.distributed.barrier()
    call_us = 1e3 * span[0].elapsed_time(span[1]) / (M * L)
    if ham.ham_kv_status(kv) != ham.HAM_DEVERR_NONE:
        raise RuntimeError("device error during the timed region")
    dprobe = capture(ham.ham_decode_step, True)       # the general step, for context
    with torch.cuda.stream(stream):
        for _ in range(3):
            dprobe.replay()
    torch.cuda.synchronize()
    decode_us = 1e3 * span[0].elapsed_time(span[1]) / (M * L)
    if ham.ham_kv_status(kv) != ham.HAM_DEVERR_NONE:
        raise RuntimeError("device error in the decode-step comparison")

    nbytes = sum(micro_call_bytes(w, C + i) for i in range(M)) / M   # per call, averaged
    peak, peak_src = measured_peak_hbm()
    value = job_throughput(steps, world, elapsed_ms * 1e-3)
    achieved = nbytes / (call_us * 1e-6) / 1e9

    # end to end: every micro-step copies its inputs for all layers (q, k, v, ntok) from pinned
    # host memory, makes the L calls and copies the L outputs back; the host reads them.  One
    # graph per micro-step position; the last also rolls the local caches back.
    hq = [[x.cpu().pin_memory() for x in row] for row in qs]
    hk = [[x.cpu().pin_memory() for x in row] for row in ks]
    hv = [[x.cpu().pin_memory() for x in row] for row in vs]
    hn = ntok.cpu().pin_memory()
    hout = [torch.empty_like(o, device="cpu").pin_memory() for o in outs]
    io = []
    for i in range(M):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            ntok.copy_(hn, non_blocking=True)
            for layer in range(L):
                qs[i][layer].copy_(hq[i][layer], non_blocking=True)
                ks[i][layer].copy_(hk[i][layer], non_blocking=True)
                vs[i][layer].copy_(hv[i][layer], non_blocking=True)
                ham.ham_micro_step(kv, layer, qs[i][layer], ks[i][layer], vs[i][layer], None,
                                   ntok, outs[layer])
                hout[layer].copy_(outs[layer], non_blocking=True)
            if i == M - 1:
                for layer in range(L):
                    ham.ham_kv_set_lengths(kv, layer, counts, tokens)
        io.append(g)
    torch.cuda.synchronize()
    n_e2e = max(M, (args.e2e_steps // M) * M)
    checksum = 0.0
    te = time.perf_counter()
    with torch.cuda.stream(stream):
        for i in range(n_e2e):
            io[i % M].replay()
            stream.synchronize()
            bits = np.uint32(np.uint16(hout[0].view(torch.int16).numpy().flat[0])) << np.uint32(16)
            checksum += float(bits.view(np.float32))
    dte = max_over_ranks(time.perf_counter() - te, world, "cuda")
    if ham.ham_kv_status(kv) != ham.HAM_DEVERR_NONE:
        raise RuntimeError("device error in the end-to-end loop")
    in_bytes = L * B * (w.n_q_heads + 2 * w.n_kv_heads) * w.head_dim * 2 + B * 4

    result = {
        "metric": MICRO_METRIC, "value": round(value, 2), "unit": "micro-steps/s",
        "n_gpus": world, "steps": steps, "warmup": n_warm * MACRO * M,
        "ms_per_step": round(elapsed_ms / steps, 5), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "accum_dtype": "f32",
        "data": "synthetic",
        "config": {"workload": w.name, "batch": B, "layers": L, "n_q_heads": w.n_q_heads,
                   "n_kv_heads": w.n_kv_heads, "head_dim": w.head_dim,
                   "context_entries": C, "micro_steps_per_macro_step": M,
                   "step": f"one micro-step: {L} ham_micro_step calls (one per layer) over "
                           f"{C}..{C + M - 1} cached entries plus the new one",
                   "graph": f"{MACRO} macro-steps per CUDA graph, each {M} micro-steps and a "
                            f"rollback of the {L} local caches to the context",
                   "l2": "local caches are L2-resident by nature (a few hundred KB)"},
        "micro_tokens_per_s": round(value * B, 1),
        "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                     "frac": round(achieved / peak, 4), "traffic": None,
                     "kernel": "micro_step_kernel", "avg_launch_us": round(call_us, 3),
                     "algorithmic_bytes_per_launch": int(nbytes), "peak_source": peak_src,
                     "note": "latency-bound: a few hundred KB per launch",
                     "duration_method": f"CUDA events around the {M * L} calls of the last "
                                        f"macro-step of the last graph replay, / {M * L}"},
        "decode_step_same_calls_us": round(decode_us, 3),
        "gpu_launches": n_graph * MACRO * (M * L + L) * world,
        "e2e": {"value": round(job_throughput(n_e2e, world, dte), 2), "unit": "micro-steps/s",
                "h2d_bytes_per_step": in_bytes,
                "d2h_bytes_per_step": L * B * w.n_q_heads * w.head_dim * 2,
                "steps": n_e2e, "finite": math.isfinite(checksum),
                "path": "every micro-step: pinned host -> device copies of each layer's q, k, v "
                        "and the token counts, one call per layer, device -> pinned host copies of "
                        "the outputs, read on the host (one CUDA graph per micro-step position)"},
        "clocks": clocks.summary(),
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        n, dt = micro_cpu_sample(w, min(args.cpu_seconds, 5.0))
        result["cpu_baseline"] = {"value": round(n / dt, 4), "unit": "micro-steps/s", "cores": 1,
                                  "kind": "oracle",
                                  "sample": f"{n} micro-steps of {w.name} (append + attention of "
                                            f"every layer, one thread)"}
    ham.ham_kv_free(kv)
    if rank == 0:
        print(json.dumps(result), flush=True)


# ---------------------------------------------------------------------------------------
# chunked prefill (prompt ingestion)
# ---------------------------------------------------------------------------------------

PREFILL_METRIC = "chunked-prefill rows/s (prompt tokens ingested per second, one layer)"


def prefill_flops(pw):
    """Algorithmic FLOPs of one call: q.k and p.v (2 multiply-adds = 4 FLOPs per element of
    head_dim) for every query head of every new row over the slots it attends."""
    w = pw.w
    n, L = pw.rows, pw.cached
    attended = n * L + n * (n + 1) // 2          # sum over rows j of (L + j + 1)
    return 4 * w.head_dim * w.n_q_heads * w.batch * attended


def prefill_bytes(pw):
    """Algorithmic bytes of one call: the K and V rows of every attended slot once per KV head
    (cached and new), q in and out, k_new / v_new in."""
    w = pw.w
    T = pw.rows * w.batch
    kv = w.batch * w.n_kv_heads * (pw.cached + pw.rows) * w.head_dim * 2 * 2
    return kv + T * w.n_q_heads * w.head_dim * 2 * 2 + T * w.n_kv_heads * w.head_dim * 2 * 2


def prefill_sample(pw, seconds, want_rows=None):
    """Rows of the chunk the CPU oracle attends in a bounded sample: evenly spread over every
    sequence's rows, so that their mean context is the chunk's."""
    per_row = 4 * pw.w.head_dim * pw.w.n_q_heads * (pw.cached + pw.rows / 2)   # fp64 FLOPs
    n = want_rows or max(8, int(seconds * 2e9 / per_row))                      # ~2 GFLOP/s
    n = min(n, pw.rows * pw.w.batch)
    import numpy as np
    idx = np.linspace(0, pw.rows * pw.w.batch - 1, n).round().astype(np.int64)
    want = np.zeros(pw.rows * pw.w.batch, bool)
    want[idx] = True
    return want


def prefill_cpu(pw, seconds):
    """The oracle as it stands on a bounded sample: every row appended, a spread sample of rows
    attended; rows/s = sampled rows / time."""
    import numpy as np

    import oracle
    from paper_2505_20438_gb300 import workload as wl
    oracle.build()
    B = pw.w.batch
    case = wl.make_prefill_case(pw.w, [pw.rows] * B, cached=np.full(B, pw.cached, np.int32))
    want = prefill_sample(pw, seconds)
    oc = oracle.OracleCache.from_case(case.base)
    q = case.q.copy()
    t0 = time.perf_counter()
    rc, _ = oc.prefill(q, case.k_new, case.v_new, case.offsets, ntok=case.ntok, want=want)
    dt = time.perf_counter() - t0
    if rc != 0:
        raise RuntimeError(f"oracle prefill failed ({rc})")
    return int(want.sum()) / dt, int(want.sum()), dt


def run_reference_prefill(args, pw):
    steps, warm = max(1, min(args.steps, 3)), 0
    vals = []
    for _ in range(steps):
        v, n, dt = prefill_cpu(pw, args.cpu_seconds / steps)
        vals.append(v)
    value = sum(vals) / len(vals)
    cores = oracle_threads()
    print(json.dumps({
        "impl": "reference", "metric": PREFILL_METRIC, "value": round(value, 3),
        "unit": "rows/s", "n_gpus": 1, "steps": steps, "warmup": warm,
        "ms_per_step": round(1e3 * pw.rows * pw.w.batch / value, 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": pw.name, "batch": pw.w.batch, "rows": pw.rows,
                   "cached": pw.cached},
        "cpu_baseline": {"value": round(value, 3), "unit": "rows/s", "cores": cores,
                         "kind": "oracle",
                         "sample": f"each step: all {pw.rows * pw.w.batch} rows appended, "
                                   f"{n} spread rows attended (fp64 C oracle, OpenMP)"},
        "e2e": {"value": round(value, 3), "unit": "rows/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }), flush=True)


def oracle_threads():
    try:
        import oracle
        return int(oracle.max_threads())
    except Exception:
        return os.cpu_count()


def run_prefill(args, pw):
    """One step = one ham_prefill call of the whole chunk (every sequence's rows: plan,
    RoPE + append, causal attention).  The counters are set back to the cached length before
    every call (one small kernel), so each step stores and attends the same slots."""
    import numpy as np
    import torch

    from paper_2505_20438_gb300 import build as build_mod
    from paper_2505_20438_gb300 import ham
    from paper_2505_20438_gb300 import workload as wl

    rank, local_rank, world = dist_env()
    torch.cuda.set_device(local_rank)
    if world > 1 and not torch.distributed.is_initialized():
        torch.distributed.init_process_group("nccl")
    build_mod.build()
    w = pw.w
    B = w.batch
    case = wl.make_prefill_case(dataclasses_replace_seed(w, rank), [pw.rows] * B,
                                cached=np.full(B, pw.cached, np.int32))
    kv = ham.ham_kv_alloc(1, B, w.n_q_heads, w.n_kv_heads, w.head_dim, w.page_slots,
                          case.base.max_slots, pool_pages=case.base.pool_pages)
    ham.ham_kv_set_page_table(kv, case.base.page_table)

    def dev(bits):
        return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(
            torch.bfloat16).cuda()

    if pw.cached:
        ham.ham_kv_fill(kv, 0, dev(case.base.k), dev(case.base.v),
                        torch.from_numpy(case.base.num_slots).cuda())
    q, k_new, v_new = dev(case.q), dev(case.k_new), dev(case.v_new)
    offsets = torch.from_numpy(case.offsets).cuda()
    ntok = torch.from_numpy(case.ntok).cuda()
    out = torch.empty_like(q)
    lens = torch.full((B,), pw.cached, dtype=torch.int32, device="cuda")
    toks = torch.full((B,), pw.cached, dtype=torch.int64, device="cuda")
    stream = torch.cuda.Stream()
    T = pw.rows * B

    def step():
        ham.ham_kv_set_lengths(kv, 0, lens, toks, stream=stream)
        ham.ham_prefill(kv, 0, q, k_new, v_new, offsets, out, ntok=ntok, stream=stream)

    steps = max(1, min(args.steps, 200))
    warm = max(3, min(args.warmup, 20))
    with torch.cuda.stream(stream):
        for _ in range(warm):
            step()
    stream.synchronize()
    if ham.ham_kv_status(kv) != ham.HAM_DEVERR_NONE:
        raise RuntimeError("device error in the warm-up")
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local_rank) as clocks, torch.cuda.stream(stream):
        t0.record(stream)
        for i in range(steps):
            if i == steps - 1:
                ham.ham_kv_set_lengths(kv, 0, lens, toks, stream=stream)
                c0.record(stream)
                ham.ham_prefill(kv, 0, q, k_new, v_new, offsets, out, ntok=ntok, stream=stream)
                c1.record(stream)
            else:
                step()
        t1.record(stream)
        torch.cuda.synchronize()
    elapsed_ms = max_over_ranks(t0.elapsed_time(t1), world, "cuda")
    if world > 1:
        torch.distributed.barrier()
    if ham.ham_kv_status(kv) != ham.HAM_DEVERR_NONE:
        raise RuntimeError("device error during the timed region")
    # the call alone, timed over a short run of calls (events around each ham_prefill)
    call_ms = []
    with torch.cuda.stream(stream):
        for _ in range(5):
            ham.ham_kv_set_lengths(kv, 0, lens, toks, stream=stream)
            c0.record(stream)
            ham.ham_prefill(kv, 0, q, k_new, v_new, offsets, out, ntok=ntok, stream=stream)
            c1.record(stream)
            c1.synchronize()
            call_ms.append(c0.elapsed_time(c1))
    call_ms = sorted(call_ms)[len(call_ms) // 2]
    flops = prefill_flops(pw)
    peak, peak_src = measured_peak_bf16()
    achieved = flops / (call_ms * 1e-3) / 1e12
    # the roofline that bounds the call: the contraction, or (a short chunk over a long cache)
    # the stream of the cached rows
    nbytes = prefill_bytes(pw)
    hbm_peak, hbm_src = measured_peak_hbm()
    gbs = nbytes / (call_ms * 1e-3) / 1e9
    hbm_bound = nbytes / hbm_peak > flops / (peak * 1e3)  # seconds x 1e9, both sides
    value = world * T * steps / (elapsed_ms * 1e-3)

    # end to end: pinned host -> device copies of the chunk's q, k, v and offsets, the call,
    # device -> pinned host copy of the output, read on the host
    hq, hk, hv = q.cpu().pin_memory(), k_new.cpu().pin_memory(), v_new.cpu().pin_memory()
    hoff = offsets.cpu().pin_memory()
    hout = torch.empty(out.shape, dtype=out.dtype).pin_memory()
    n_e2e = max(3, min(args.e2e_steps, 20))
    checksum = 0.0
    te = time.perf_counter()
    with torch.cuda.stream(stream):
        for _ in range(n_e2e):
            q.copy_(hq, non_blocking=True)
            k_new.copy_(hk, non_blocking=True)
            v_new.copy_(hv, non_blocking=True)
            offsets.copy_(hoff, non_blocking=True)
            ham.ham_kv_set_lengths(kv, 0, lens, toks, stream=stream)
            ham.ham_prefill(kv, 0, q, k_new, v_new, offsets, out, ntok=ntok, stream=stream)
            hout.copy_(out, non_blocking=True)
            stream.synchronize()
            checksum += float(hout[0, 0, 0])
    dte = max_over_ranks(time.perf_counter() - te, world, "cuda")
    h2d = sum(t.numel() * t.element_size() for t in (q, k_new, v_new, offsets))
    result = {
        "metric": PREFILL_METRIC, "value": round(value, 1), "unit": "rows/s", "n_gpus": world,
        "steps": steps, "warmup": warm, "ms_per_step": round(elapsed_ms / steps, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "accum_dtype": "f32", "data": "synthetic",
        "config": {"workload": pw.name, "batch": B, "rows_per_sequence": pw.rows,
                   "cached_slots": pw.cached, "n_q_heads": w.n_q_heads,
                   "n_kv_heads": w.n_kv_heads, "head_dim": w.head_dim,
                   "page_slots": w.page_slots, "tokens_per_row": 1,
                   "step": "ham_kv_set_lengths + ham_prefill (plan, RoPE + append, causal "
                           "attention) of the whole chunk",
                   "l2": ("inputs larger than L2 (q, out 134 MB each at the 4 x 4096 chunk)"
                          if pw.rows * B >= 4096 else
                          f"cached K and V ({prefill_bytes(pw) / 2**20:.0f} MiB) larger than L2")},
        "tflops": round(achieved, 1),
        "roofline": dict(
            ({"bound": "hbm", "achieved": round(gbs, 1), "peak": hbm_peak, "unit": "GB/s",
              "frac": round(gbs / hbm_peak, 4), "algorithmic_bytes_per_launch": int(nbytes),
              "peak_source": hbm_src, "tensor_frac_of_measured": round(achieved / peak, 4)}
             if hbm_bound else
             {"bound": "tensor", "achieved": round(achieved, 1), "peak": peak,
              "unit": "TFLOP/s", "frac": round(achieved / peak, 4),
              "algorithmic_flops_per_launch": int(flops), "peak_source": peak_src,
              "hbm_frac_of_measured": round(gbs / hbm_peak, 4)}),
            traffic=None,
            kernel="prefill_attn_kernel (with the plan, RoPE + append and, when the grid "
                   "splits over the cached slots, merge kernels of the same call)",
            avg_launch_us=round(call_ms * 1e3, 1),
            duration_method="CUDA events around one ham_prefill call, median of 5"),
        "gpu_launches": steps * 4 * world,
        "e2e": {"value": round(world * T * n_e2e / dte, 1), "unit": "rows/s",
                "h2d_bytes_per_step": int(h2d),
                "d2h_bytes_per_step": int(out.numel() * out.element_size()),
                "steps": n_e2e, "finite": math.isfinite(checksum),
                "path": "every step: pinned host -> device copies of q, k, v and offsets, "
                        "ham_prefill, device -> pinned host copy of the output"},
        "clocks": clocks.summary(),
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        v, n, dt = prefill_cpu(pw, args.cpu_seconds)
        result["cpu_baseline"] = {
            "value": round(v, 3), "unit": "rows/s", "cores": oracle_threads(), "kind": "oracle",
            "sample": f"all {T} rows appended, {n} spread rows attended in {dt:.1f} s (fp64 C "
                      f"oracle, OpenMP)"}
    ham.ham_kv_free(kv)
    if rank == 0:
        print(json.dumps(result), flush=True)


def dataclasses_replace_seed(w, rank):
    """Rank r's sequences: the workload's seed shifted by the rank (ranks own different
    sequences)."""
    import dataclasses
    return dataclasses.replace(w, seed=w.seed + 100 * rank)


def main():
    global CACHES
    args = parse_args()
    if args.caches < 1 or GRAPH_STEPS % args.caches:
        raise SystemExit(f"--caches must divide {GRAPH_STEPS}")
    CACHES = args.caches
    w = workload(args.workload)
    from paper_2505_20438_gb300 import workload as wl
    if args.impl == "reference":
        return run_reference(args, w)
    import torch
    if not torch.cuda.is_available():
        raise SystemExit("bench.py: this arm runs the library's CUDA kernels and needs a GPU "
                         "(GB300); there is no CPU path (--impl reference times the oracle)")
    if isinstance(w, wl.EmbedWorkload):
        run_embed(args, w)
    elif isinstance(w, wl.FrontWorkload):
        run_front(args, w)
    elif isinstance(w, wl.MicroWorkload):
        run_micro(args, w)
    elif isinstance(w, wl.PrefillWorkload):
        run_prefill(args, w)
    elif w.layers > 1:
        run_stack(args, w)
    else:
        run_ours(args, w)


if __name__ == "__main__":
    main()
