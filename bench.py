#!/usr/bin/env python3
"""Benchmark of the GEMV-bound decode chain (one JSON line on rank 0).

Workload (the headline): the 3B-shaped decode chain at batch 1 -- 28 layers of
fused QKV (5120 x 3072), O (3072 x 3072), gate_up (16384 x 3072) and down
(3072 x 8192) projections plus the LM head (128256 x 3072), int4 codes in
groups of 32 with fp16 scales (1.807 GB per token), seeded synthetic weights
resident in HBM.  One step = one decoded token = one launch of the persistent
chain kernel through wq4_decode_chain.  The weights (1.8 GB) are far larger
than L2 (129 MB), so no L2 flush is needed between steps.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--workload 3b|8b|phi3.5] [--batch B]
    python bench.py --workload attn-8b|attn-3b|attn-8b-b1     (decode attention)
    python bench.py --workload prefill-3b [--tokens M]         (prefill-shaped GEMMs)
    python bench.py --workload gemv-2048|gemv-3b-layer         (single wq4_gemv calls)

The attn-* workloads time decode attention of one layer over a paged
key/value cache instead (wq4_paged_attention, one launch per step): 32
sequences with context lengths uniform on [1, 8192] (attn-8b-b1: one
sequence of 4096), Llama-3.1-8B- or 3B-shaped heads, pages of 16 tokens.

--impl reference times the fp64 CPU oracle on a bounded sample of the same
workload (the only reference this repository has: the paper's WebGPU/Metal
engine cannot run here).  Under torchrun (N > 1) every rank decodes its own
replica (no collective: the workload does not exchange data between GPUs).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "GEMV-bound decode tokens/s (batch 1) and achieved HBM GB/s vs ~8 TB/s peak"
NOMINAL_HBM_GBS = 8000.0
# the paper's batch-1 decode rates for these model shapes (Table 1, WebLLM in
# Chrome on an Apple M3 Max, 4-bit weights): another machine's numbers, context only
PAPER_DECODE_TOKS = {"8b": 41.1, "phi3.5": 71.1}
# rotary base of the model families the shapes follow (Llama-3.x, Phi-3.5)
ROPE_THETA = {"3b": 500000.0, "8b": 500000.0, "phi3.5": 10000.0}
FALLBACK_HBM_GBS = 6800.0
L2_BYTES = 129 * 1024 * 1024


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=["3b", "8b", "phi3.5", "attn-8b", "attn-3b", "attn-8b-b1", "prefill-3b",
                                           "gemv-2048", "gemv-3b-layer"],
                    default="3b")
    ap.add_argument("--tokens", type=int, default=2048, help="prompt tokens of the prefill workload")
    ap.add_argument("--batch", type=int, default=1)
    ap.add_argument("--layers", type=int, default=0, help="override the layer count (profiling runs)")
    ap.add_argument("--context", type=int, default=0,
                    help="decode step with attention (wq4_decode_step) at this many tokens of context "
                         "(0: the GEMV-bound chain with the query-block stand-in)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    return ap.parse_args()


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def measured_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        d = json.load(open(path))
        return float(d["hbm_gbs"]), "measured (MEASURED_PEAKS.json hbm_gbs, copy read+write)"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


KERNEL_SOURCES = {
    "chain_kernel": ("wq4_chain.cu", "wq4_items.cuh", "wq4_device.cuh"),
    "tc_stage_kernel": ("wq4_tc.cu", "wq4_tc.cuh", "wq4_device.cuh"),
}


def chain_source_sha(kernel: str) -> str:
    """Hash of the sources of one kernel (the committed ncu summary of that
    kernel carries the same hash)."""
    h = hashlib.sha256()
    for f in KERNEL_SOURCES[kernel]:
        h.update(open(os.path.join(ROOT, "paper_2412_15803_gb300", "csrc", f), "rb").read())
    return h.hexdigest()[:16]


def profiled_traffic(name: str, workload: str, batch: int, context: int = 0):
    """DRAM bytes per launch of kernel `name` from the committed ncu summary,
    if it was taken on the current kernel source (else None)."""
    ctx = f"_ctx{context}" if context else ""
    path = os.path.join(ROOT, "profiles", f"{name}_{workload}_b{batch}{ctx}.md")
    if not os.path.exists(path):
        return None
    text = open(path).read()
    m = re.search(r"traffic_bytes_per_launch:\s*(\d+)", text)
    s = re.search(r"source_sha:\s*([0-9a-f]+)", text)
    if not m or not s or s.group(1) != chain_source_sha(name):
        return None
    return int(m.group(1))


class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.proc = None
        self.out = None
        try:
            import torch
            uuid = str(torch.cuda.get_device_properties(device_index).uuid)
            sel = ["-i", uuid if uuid.startswith("GPU-") else "GPU-" + uuid]
        except Exception:
            sel = []
        self.cmd = ["nvidia-smi", *sel, f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "100"]

    def start(self):
        try:
            self.proc = subprocess.Popen(self.cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, mx, reasons, power = [], [], set(), []
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [t.strip() for t in line.split(",")]
            if len(f) < 8:
                continue
            try:
                sm.append(float(f[0]))
                mx.append(float(f[1]))
                power.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm),
                "power_w_median": statistics.median(power) if power else None}


# ---------------------------------------------------------------- oracle --

def host_info() -> dict:
    """The host the CPU baselines ran on: cores this process may use, CPU model."""
    import platform
    try:
        nproc = len(os.sched_getaffinity(0))
    except Exception:
        nproc = os.cpu_count() or 1
    model = None
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().lower().startswith("model name"):
                model = line.split(":", 1)[1].strip()
                break
    except Exception:
        pass
    if not model:
        try:
            with open("/proc/cpuinfo") as f:
                for line in f:
                    if line.lower().startswith("model name"):
                        model = line.split(":", 1)[1].strip()
                        break
        except Exception:
            pass
    return {"nproc": nproc, "cpu_model": model or "unknown", "machine": platform.machine()}


class RowPool:
    """Runs the oracle's GEMV over row blocks on `threads` threads.  The C
    routine releases the GIL, so the blocks run on separate cores; every row
    is computed by the same code as in a single call."""

    def __init__(self, threads: int):
        from concurrent.futures import ThreadPoolExecutor
        self.threads = max(1, threads)
        self.ex = ThreadPoolExecutor(self.threads) if self.threads > 1 else None

    def gemv(self, W, s, x):
        import oracle
        N = W.shape[0]
        if self.ex is None or N < 2 * self.threads:
            oracle.gemv(W, s, x)
            return
        cuts = [N * i // self.threads for i in range(self.threads + 1)]
        list(self.ex.map(lambda i: oracle.gemv(W[cuts[i]:cuts[i + 1]], s[cuts[i]:cuts[i + 1]], x),
                         range(self.threads)))

    def close(self):
        if self.ex is not None:
            self.ex.shutdown()


def oracle_sample(shape, batch: int, fraction: float, seed: int = 0, pool: RowPool | None = None):
    """Times the fp64 oracle on the first ceil(fraction * N) rows of every
    projection of the chain (all layers and the LM head); with a pool, each
    block's rows are split over its threads.  Returns (seconds, weights
    processed)."""
    import oracle
    from paper_2412_15803_gb300 import synth
    x = {K: synth.activations(seed, batch, K) for K in {shape.hidden, shape.ffn}}
    blocks = []
    for l in range(shape.num_layers):
        for name, N, K, mat in shape.mats(l):
            blocks.append((N, K, l, mat))
    blocks.append((shape.vocab, shape.hidden, shape.num_layers, synth.MAT_LM_HEAD))
    total_t, total_w = 0.0, 0
    for N, K, l, mat in blocks:
        n = max(1, int(np.ceil(fraction * N)))
        W, s = synth.matrix(seed, N, K, l, mat, 0, n, symmetric=True)
        t0 = time.perf_counter()
        if pool is None:
            oracle.gemv(W, s, x[K])
        else:
            pool.gemv(W, s, x[K])
        total_t += time.perf_counter() - t0
        total_w += n * K
    return total_t, total_w


def oracle_rate_estimate(shape, batch):
    """Seconds per weight of the oracle on this host (short calibration)."""
    import oracle
    from paper_2412_15803_gb300 import synth
    W, s = synth.matrix(1, 256, shape.hidden)
    x = synth.activations(1, batch, shape.hidden)
    t0 = time.perf_counter()
    oracle.gemv(W, s, x)
    return (time.perf_counter() - t0) / (256 * shape.hidden)


def all_core_line(value: float, unit: str, threads: int, sample: str) -> dict:
    return {"value": value, "unit": unit, "cores": threads,
            "kind": f"oracle, row-parallel: the same fp64 C routine over {threads} row blocks on {threads} threads",
            "sample": sample}


def oracle_attention_layer_s(shape, batch: int, context: int, seed: int = 0) -> float:
    """Seconds of the fp64 oracle's paged attention for one layer of a decode
    step: every row attends to `context` tokens of a seeded paged cache."""
    import oracle
    from paper_2412_15803_gb300 import synth
    P, D = 16, shape.head_dim
    lens = np.full(batch, context, np.int32)
    num_pages = int(((lens + P - 1) // P).sum())
    table = synth.page_table(seed, lens, P, num_pages)
    k, v = synth.kv_cache(seed, num_pages, shape.n_kv_heads, P, D)
    q = synth.queries(seed, batch, shape.n_q_heads, D)
    t0 = time.perf_counter()
    oracle.paged_attention(q, k, v, table, lens, 1.0 / np.sqrt(D), shape.n_q_heads)
    return time.perf_counter() - t0


def cpu_baseline(shape, batch, target_s=12.0, context: int = 0):
    per_w = oracle_rate_estimate(shape, batch)
    frac = min(1.0, target_s / max(per_w * shape.weight_count(), 1e-9))
    t, w = oracle_sample(shape, batch, frac)
    tokens = batch * w / shape.weight_count()
    host = host_info()
    pool = RowPool(host["nproc"])
    tp, wp = oracle_sample(shape, batch, frac, pool=pool)
    pool.close()
    line = {"value": tokens / t, "unit": "tokens/s", "cores": 1, "kind": "oracle",
            "sample": f"first {frac:.4f} of the rows of all {4 * shape.num_layers + 1} projections "
                      f"({w} weights = {w / shape.weight_count():.4f} of a token), batch {batch}, "
                      f"single-threaded fp64 C oracle, {t:.1f} s",
            **host,
            "all_core": all_core_line(batch * wp / shape.weight_count() / tp, "tokens/s", pool.threads,
                                      f"the same rows, {tp:.1f} s")}
    if context:
        # a step adds every layer's attention: timed on one layer, counted L times
        ta = oracle_attention_layer_s(shape, batch, context)
        step_s = t * shape.weight_count() / w + shape.num_layers * ta
        line["value"] = batch / step_s
        line["sample"] += (f"; plus the oracle's attention of one layer over {context} tokens x {batch} rows "
                           f"({ta:.2f} s), counted for all {shape.num_layers} layers")
        step_p = tp * shape.weight_count() / wp + shape.num_layers * ta
        line["all_core"]["value"] = batch / step_p
        line["all_core"]["sample"] += " (the attention single-threaded)"
    return line


def chain_step_bytes(shape, B: int) -> int:
    """Bytes one token step streams: packed codes + scales of every
    projection, plus the activation vectors read and written (negligible)."""
    return shape.weight_bytes() + 2 * B * (shape.hidden * (4 * shape.num_layers + 1) + shape.vocab)


def chain_config(shape, B: int, world: int, context: int = 0) -> dict:
    """The workload's config object, the same for both arms."""
    what = "decode chain" if not context else \
        f"decode step with attention ({shape.n_q_heads} q / {shape.n_kv_heads} kv heads of {shape.head_dim}, " \
        f"RoPE, paged KV cache of 16-token pages, {context} tokens of context per row)"
    kv = 0 if not context else context - 1
    kv_bytes = B * kv * shape.n_kv_heads * shape.head_dim * 2 * 2 * shape.num_layers
    return {"workload": f"{shape.name}-shaped {what}: {shape.num_layers} layers x "
                        f"(QKV {shape.n_qkv}x{shape.hidden}, O {shape.hidden}x{shape.hidden}, "
                        f"gate_up {2 * shape.ffn}x{shape.hidden}, down {shape.hidden}x{shape.ffn}) "
                        f"+ LM head {shape.vocab}x{shape.hidden}, batch {B}",
            "batch": B, "context": context, "bytes_per_token": chain_step_bytes(shape, B) + kv_bytes,
            "l2": "inputs larger than L2 (1.8+ GB of weights per step), no flush",
            "codes": "drawn uniform on 0..14 (zero-mean q - 7), not 0..15: with 0..15 the mean offset of "
                     "+0.5 per weight compounds through 28-32 layers and overflows fp16 in the oracle's own "
                     "chain; the kernels' work and timing do not depend on the code values, and every code "
                     "value 0..15 runs through the chain in the full-range parity tests",
            "parallelism": "replicas" if world > 1 else "single GPU"}


def run_reference(args, rank, world):
    from paper_2412_15803_gb300.model import SHAPES
    if rank != 0:
        return
    shape = SHAPES[args.workload]
    T = args.context
    per_w = oracle_rate_estimate(shape, args.batch)
    nsteps = args.steps + args.warmup
    step_s = min(10.0, 120.0 / max(nsteps, 1))
    frac = min(1.0, step_s / (per_w * shape.weight_count()))
    # with attention, one layer's attention is timed once per step as well
    times, wsum, atimes = [], 0, []
    for i in range(nsteps):
        t, w = oracle_sample(shape, args.batch, frac)
        a = oracle_attention_layer_s(shape, args.batch, T, seed=i) if T and i >= args.warmup else 0.0
        if i >= args.warmup:
            times.append(t)
            atimes.append(a)
            wsum += w
    steps = len(times)
    token_s = sum(times) * shape.weight_count() / wsum + shape.num_layers * (sum(atimes) / steps if T else 0.0)
    value = args.batch / token_s
    sample = (f"each step: first {frac:.5f} of the rows of every projection "
              f"(all {4 * shape.num_layers + 1}), scaled to a token by weights")
    if T:
        sample += f"; plus one layer's attention over {T} tokens, counted for all {shape.num_layers} layers"
    line = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * token_s, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded SplitMix64 weights and activations)", "impl": "reference",
            "config": chain_config(shape, args.batch, world, T),
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": 1, "kind": "oracle", "sample": sample,
                             **host_info()},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------- ours --

def aggregate_replicas(total_ms: float, e2e_s_per_step: float, batch: int, steps: int, device="cpu"):
    """Whole-job numbers over the ranks of the default process group (if any).

    Every rank decodes its own replica for the same number of steps, so the
    job time is the slowest rank's: returns (tokens/s, e2e tokens/s, job ms)
    computed from the MAX over ranks of the timed region and of the e2e time
    per step.  Works with any backend (nccl on GPUs, gloo on CPU)."""
    import torch
    import torch.distributed as dist
    world = dist.get_world_size() if dist.is_available() and dist.is_initialized() else 1
    t = torch.tensor([total_ms, e2e_s_per_step], dtype=torch.float64, device=device)
    if world > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    job_ms, e2e_step = float(t[0].item()), float(t[1].item())
    return world * batch * steps / (job_ms / 1e3), world * batch / e2e_step, job_ms


def run_ours(args, rank, world, local):
    import torch
    import torch.distributed as dist
    from paper_2412_15803_gb300 import synth, wq4
    from paper_2412_15803_gb300.model import SHAPES, DecodeModel, StepCaches

    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    shape = SHAPES[args.workload]
    if args.layers:
        import dataclasses
        shape = dataclasses.replace(shape, name=f"{shape.name}-{args.layers}l", num_layers=args.layers)
    B = args.batch
    T = args.context
    model = DecodeModel(shape, batch=B, seed=0, step=T > 0)
    x_np = synth.activations(1000 + rank, B, shape.hidden)
    x = torch.from_numpy(x_np.view(np.int16)).cuda()
    logits = torch.empty((B, shape.vocab), dtype=torch.int16, device="cuda")
    stream = torch.cuda.current_stream()

    step_bytes = chain_step_bytes(shape, B)
    if T > 0:
        # every row decodes the token at position T - 1: it attends to T tokens
        caches = StepCaches(shape, [T - 1] * B, seed=1, rope_theta=ROPE_THETA.get(args.workload, 500000.0))
        step_bytes += caches.cache_bytes_read()

        def decode():
            model.decode_step(caches, x, logits, stream)

        def decode_host(xh, lh):
            model.decode_step_host(caches, xh, lh, stream)
    else:
        def decode():
            model.decode(x, logits, stream)

        def decode_host(xh, lh):
            model.decode_host(xh, lh, stream)

    for _ in range(args.warmup):
        decode()
    torch.cuda.synchronize()
    if wq4.wq4_device_status(stream) != 0:
        raise RuntimeError("device wait timed out during warm-up")
    # the library's choice for this table: the persistent chain kernel, or the
    # stage graph (batches above its limit, or a ring that does not fit)
    persistent = wq4.wq4_chain_path(model.table, decode_step=T > 0) == 1

    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.3)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    for i in range(args.steps):
        starts[i].record(stream)
        decode()
        ends[i].record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clocks = sampler.stop()
    total_ms = starts[0].elapsed_time(ends[-1])
    launch_ms = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    if wq4.wq4_device_status(stream) != 0:
        raise RuntimeError("device wait timed out during the timed region")

    # end to end through the host-buffer entry point: x H2D, chain, logits D2H
    x_host = torch.from_numpy(x_np.view(np.int16)).pin_memory()
    l_host = torch.empty((B, shape.vocab), dtype=torch.int16).pin_memory()
    e2e_steps = max(10, min(args.steps, 500))
    for _ in range(3):
        decode_host(x_host.numpy(), l_host.numpy())
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        decode_host(x_host.numpy(), l_host.numpy())
    e2e_s = time.perf_counter() - t0
    tokens_per_s, e2e_val, total_ms_max = aggregate_replicas(total_ms, e2e_s / e2e_steps, B, args.steps, "cuda")

    if persistent:
        # one cooperative launch of the persistent chain kernel per token
        kernel_name, launches_per_step = "chain_kernel", 1
    else:
        # one CUDA-graph replay: a prologue and one tensor-core stage kernel per
        # projection (with attention, three more a layer: rotation/append,
        # paged attention, the O input's token-start kernel)
        kernel_name, launches_per_step = "tc_stage_kernel", 4 * shape.num_layers + 2 + (3 * shape.num_layers if T else 0)
    if rank == 0:
        ms = total_ms_max / args.steps
        avg_launch_ms = statistics.mean(launch_ms)
        peak, peak_src = measured_peak()
        achieved = step_bytes / (avg_launch_ms * 1e-3) / 1e9
        line = {
            "metric": METRIC, "value": tokens_per_s, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak",
            "vs_baseline": (tokens_per_s / PAPER_DECODE_TOKS[args.workload]
                            if B == 1 and args.workload in PAPER_DECODE_TOKS and not args.layers and not T
                            else None),
            "dtype": "f32",
            "precision": "int4 codes (group 32, fp16 scale, zero point 7), fp16 activations, fp32 accumulation",
            "data": "synthetic (seeded SplitMix64 weights and activations)",
            "config": chain_config(shape, B, world, T),
            "hbm_gbs": step_bytes * args.steps / (total_ms_max / 1e3) / 1e9,
            "hbm_frac_of_nominal_8tbs": step_bytes * args.steps / (total_ms_max / 1e3) / 1e9 / NOMINAL_HBM_GBS,
            "roofline": {"bound": "hbm", "kernel": kernel_name, "achieved": achieved, "peak": peak,
                         "peak_source": peak_src, "unit": "GB/s", "frac": achieved / peak,
                         "frac_of_nominal_8tbs": achieved / NOMINAL_HBM_GBS,
                         "traffic": profiled_traffic(kernel_name, args.workload, B, T),
                         "algorithmic_bytes_per_launch": step_bytes,
                         "avg_launch_ms": avg_launch_ms},
            "e2e": {"value": e2e_val, "unit": "tokens/s", "h2d_bytes_per_step": 2 * B * shape.hidden,
                    "d2h_bytes_per_step": 2 * B * shape.vocab},
            "gpu_launches": args.steps * launches_per_step,
            "clocks": clocks,
        }
        if line["vs_baseline"] is not None:
            line["vs_baseline_ref"] = (f"paper Table 1: {PAPER_DECODE_TOKS[args.workload]} tok/s, WebLLM on an Apple "
                                       "M3 Max (other hardware, trained weights)")
        if world == 1 and not args.no_cpu_baseline:
            line["cpu_baseline"] = cpu_baseline(shape, B, context=T)
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


# ------------------------------------------------------------------ gemv --

# Single wq4_gemv calls: one 2048 x 2048 matrix, and the four projections of
# one 3B-shaped layer, at batch 1; codes uniform on 0..15, scales uniform on
# [0.005, 0.02], x ~ N(0, 1), seed 0 (copy 0 of the rotation is exactly that
# matrix set; copy c draws the streams of layer c).
GEMV_WORKLOADS = {
    "gemv-2048": [("gemv", 2048, 2048)],
    "gemv-3b-layer": [("qkv", 5120, 3072), ("o", 3072, 3072), ("gate_up", 16384, 3072), ("down", 3072, 8192)],
}


def gemv_set_bytes(mats) -> int:
    """Algorithmic bytes of one pass over the set: packed codes + scales
    (the activations, 2 B per K and N, are added separately)."""
    return sum(N * K // 2 + N * K // 16 for _, N, K in mats)


def gemv_copies(mats) -> int:
    """Copies of the set in rotation: together more than 4x L2."""
    return -(-4 * L2_BYTES // gemv_set_bytes(mats)) + 1


def gemv_kernel_names(mats, B: int) -> str:
    """The kernels wq4_gemv's size rule picks for the set (batch 1-2, K % 256 == 0)."""
    names = []
    for _, N, K in mats:
        k = "gemv_mma_kernel" if B <= 2 and K % 256 == 0 and N * K >= 12 << 20 else "gemv_tma_kernel"
        if k not in names:
            names.append(k)
    return "+".join(names)


def gemv_io_bytes(mats, B: int) -> int:
    return sum(2 * B * (N + K) for _, N, K in mats)


def gemv_source_sha() -> str:
    h = hashlib.sha256()
    for f in ("wq4_gemv.cu", "wq4_items.cuh", "wq4_device.cuh"):
        h.update(open(os.path.join(ROOT, "paper_2412_15803_gb300", "csrc", f), "rb").read())
    return h.hexdigest()[:16]


def gemv_profiled_traffic(workload: str):
    path = os.path.join(ROOT, "profiles", f"gemv_kernels_{workload}.md")
    if not os.path.exists(path):
        return None
    text = open(path).read()
    m = re.search(r"traffic_bytes_per_set:\s*(\d+)", text)
    h = re.search(r"source_sha:\s*([0-9a-f]+)", text)
    if not m or not h or h.group(1) != gemv_source_sha():
        return None
    return int(m.group(1))


def gemv_config(workload: str, mats, B: int, copies: int) -> dict:
    desc = ", ".join(f"{n} {N}x{K}" for n, N, K in mats)
    return {"workload": f"{workload}: wq4_gemv at batch {B} ({desc}), one launch per matrix",
            "batch": B, "bytes_per_set": gemv_set_bytes(mats) + gemv_io_bytes(mats, B),
            "codes": "uniform on 0..15", "scales": "uniform on [0.005, 0.02]", "x": "N(0, 1) fp16",
            "l2": f"{copies} copies of the set in rotation ({copies * gemv_set_bytes(mats) / 1e6:.0f} MB, more "
                  "than 4x L2), one CUDA graph replay runs every copy once",
            "parallelism": "single GPU"}


def gemv_oracle_step(mats, B: int, step_s: float, pool: RowPool | None = None):
    """The oracle on the first rows of every matrix of the set, sized to about
    step_s seconds.  Returns (seconds, bytes of weights processed)."""
    import oracle
    from paper_2412_15803_gb300 import synth
    W, sc = synth.matrix(0, 64, mats[0][2])
    x = synth.activations(0, B, mats[0][2])
    t0 = time.perf_counter()
    oracle.gemv(W, sc, x)
    per_w = (time.perf_counter() - t0) / (64 * mats[0][2])
    total_w = sum(N * K for _, N, K in mats)
    est = max(per_w * total_w, 1e-9)           # seconds of one whole set
    frac = min(1.0, step_s / est)
    reps = max(1, int(step_s / est)) if frac >= 1.0 else 1
    t, nbytes = 0.0, 0
    for i, (_, N, K) in enumerate(mats):
        n = max(1, int(np.ceil(frac * N)))
        W, sc = synth.matrix(0, N, K, 0, i, 0, n)
        x = synth.activations(0, B, K)
        t0 = time.perf_counter()
        for _ in range(reps):
            if pool is None:
                oracle.gemv(W, sc, x)
            else:
                pool.gemv(W, sc, x)
        t += time.perf_counter() - t0
        nbytes += reps * (n * K // 2 + n * K // 16)
    what = f"{reps} passes over every matrix" if reps > 1 or frac >= 1.0 else \
        f"first {frac:.4f} of the rows of every matrix"
    return t, nbytes, what


def run_gemv_reference(args, rank, world):
    if rank != 0:
        return
    mats = GEMV_WORKLOADS[args.workload]
    B = args.batch
    nsteps = args.steps + args.warmup
    step_s = min(5.0, 120.0 / max(nsteps, 1))
    times, nb, what = [], 0, ""
    for i in range(nsteps):
        t, b, what = gemv_oracle_step(mats, B, step_s)
        if i >= args.warmup:
            times.append(t)
            nb += b
    value = nb / sum(times) / 1e9
    copies = gemv_copies(mats)
    step_b = copies * (gemv_set_bytes(mats) + gemv_io_bytes(mats, B))
    line = {"metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * step_b / (value * 1e9), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded SplitMix64 weights and activations)", "impl": "reference",
            "config": gemv_config(args.workload, mats, B, copies),
            "cpu_baseline": {"value": value, "unit": "GB/s", "cores": 1, "kind": "oracle",
                             "sample": f"each step: {what}, single-threaded fp64 C oracle; ms_per_step "
                                       f"scales its rate to the {copies} sets of one step",
                             **host_info()},
            "e2e": {"value": value, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_gemv(args, rank, world, local):
    import torch
    import torch.distributed as dist
    from paper_2412_15803_gb300 import synth, wq4
    from paper_2412_15803_gb300.model import fill_matrix

    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    mats = GEMV_WORKLOADS[args.workload]
    B = args.batch
    set_b = gemv_set_bytes(mats)
    io_b = gemv_io_bytes(mats, B)
    copies = gemv_copies(mats)
    weights = []
    for c in range(copies):
        ws = []
        for i, (_, N, K) in enumerate(mats):
            W = torch.empty((N, K // 8), dtype=torch.int32, device="cuda")
            sc = torch.empty((N, K // 32), dtype=torch.int16, device="cuda")
            fill_matrix(W, sc, N, K, 0, c, i, symmetric=False)
            ws.append((W, sc))
        weights.append(ws)
    xs = {K: torch.from_numpy(synth.activations(0, B, K).view(np.int16)).cuda() for _, _, K in mats}
    ys = [torch.empty((B, N), dtype=torch.int16, device="cuda") for _, N, _ in mats]

    def one_set(c, stream):
        for i, (_, N, K) in enumerate(mats):
            W, sc = weights[c][i]
            wq4.wq4_gemv(W, sc, xs[K], ys[i], N, K, B, stream)

    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        one_set(0, stream)
        stream.synchronize()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=stream):
            for c in range(copies):
                one_set(c, stream)
        for _ in range(max(args.warmup, 3)):
            graph.replay()
    torch.cuda.synchronize()
    if wq4.wq4_device_status(stream) != 0:
        raise RuntimeError("device flag set during warm-up")

    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.3)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        for i in range(args.steps):
            starts[i].record(stream)
            graph.replay()
            ends[i].record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clocks = sampler.stop()
    total_ms = starts[0].elapsed_time(ends[-1])
    replay_ms = [s.elapsed_time(e) for s, e in zip(starts, ends)]

    # single-set latency, one launch per matrix from a cold L2 (a 2x L2 buffer
    # is written before each), and the same warm (the set just ran)
    flush = torch.empty(2 * L2_BYTES, dtype=torch.uint8, device="cuda")
    cold, warm = [], []
    with torch.cuda.stream(stream):
        for rep in range(20):
            flush.fill_(rep & 0xFF)
            e0, e1, e2 = (torch.cuda.Event(enable_timing=True) for _ in range(3))
            e0.record(stream)
            one_set(0, stream)
            e1.record(stream)
            one_set(0, stream)
            e2.record(stream)
            stream.synchronize()
            cold.append(e0.elapsed_time(e1))
            warm.append(e1.elapsed_time(e2))
    del flush

    # end to end through the C ABI call: x from pinned host memory, the set's
    # GEMVs, y back to pinned host memory, every step
    x_host = {K: v.cpu().pin_memory() for K, v in xs.items()}
    y_host = [torch.empty_like(y, device="cpu").pin_memory() for y in ys]
    e2e_steps = max(20, min(args.steps * copies, 2000))
    with torch.cuda.stream(stream):
        for i in range(e2e_steps + 5):
            if i == 5:
                t0 = time.perf_counter()
            for K, v in xs.items():
                v.copy_(x_host[K], non_blocking=True)
            one_set(i % copies, stream)
            for y, yh in zip(ys, y_host):
                yh.copy_(y, non_blocking=True)
            stream.synchronize()
        e2e_s = (time.perf_counter() - t0) / e2e_steps
    if wq4.wq4_device_status(stream) != 0:
        raise RuntimeError("device flag set during the timed region")
    t = torch.tensor([total_ms, e2e_s], dtype=torch.float64, device="cuda")
    if world > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    job_ms, e2e_step = float(t[0]), float(t[1])
    if rank == 0:
        peak, src = measured_peak()
        per_set_ms = statistics.mean(replay_ms) / copies
        step_bytes = set_b + io_b
        achieved = step_bytes / (per_set_ms * 1e-3) / 1e9
        traffic = gemv_profiled_traffic(args.workload)
        line = {
            "metric": METRIC, "value": world * step_bytes * copies * args.steps / (job_ms * 1e-3) / 1e9,
            "unit": "GB/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": job_ms / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32",
            "precision": "int4 codes (group 32, fp16 scale, zero point 7), fp16 activations, fp32 accumulation",
            "data": "synthetic (seeded SplitMix64 weights and activations)",
            "config": gemv_config(args.workload, mats, B, copies),
            "step": f"one CUDA graph replay: {copies} sets x {len(mats)} launches",
            "per_set_us": per_set_ms * 1e3,
            "per_launch_us": per_set_ms * 1e3 / len(mats),
            "single_set_latency_us": {"cold_l2_median": 1e3 * statistics.median(cold),
                                      "warm_l2_median": 1e3 * statistics.median(warm),
                                      "launches": len(mats)},
            "hbm_frac_of_nominal_8tbs": achieved / NOMINAL_HBM_GBS,
            "roofline": {"bound": "hbm", "kernel": gemv_kernel_names(mats, B), "achieved": achieved, "peak": peak,
                         "peak_source": src, "unit": "GB/s", "frac": achieved / peak,
                         "traffic": traffic, "traffic_unit": "bytes per set (ncu, cold L2)",
                         "algorithmic_bytes_per_set": step_bytes, "avg_set_ms": per_set_ms},
            "e2e": {"value": step_bytes / e2e_step / 1e9, "unit": "GB/s",
                    "h2d_bytes_per_step": sum(2 * B * K for K in xs),
                    "d2h_bytes_per_step": sum(2 * B * N for _, N, _ in mats),
                    "step": "one set through wq4_gemv with host copies"},
            "gpu_launches": args.steps * copies * len(mats),
            "clocks": clocks,
        }
        if world == 1 and not args.no_cpu_baseline:
            t1, b1, what = gemv_oracle_step(mats, B, 10.0)
            host = host_info()
            pool = RowPool(host["nproc"])
            tp, bp, what_p = gemv_oracle_step(mats, B, 10.0 * min(pool.threads, 8), pool)
            pool.close()
            line["cpu_baseline"] = {
                "value": b1 / t1 / 1e9, "unit": "GB/s", "cores": 1, "kind": "oracle",
                "sample": f"{what}, single-threaded fp64 C oracle, {t1:.1f} s",
                **host,
                "all_core": all_core_line(bp / tp / 1e9, "GB/s", pool.threads,
                                          f"{what_p}, {tp:.1f} s")}
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


# -------------------------------------------------------------- attention --

ATTN_METRIC = "paged decode attention sequences/s (one decode step per sequence) and achieved HBM GB/s"


def attn_source_sha() -> str:
    h = hashlib.sha256()
    for f in ("wq4_attn.cu", "wq4_device.cuh"):
        h.update(open(os.path.join(ROOT, "paper_2412_15803_gb300", "csrc", f), "rb").read())
    return h.hexdigest()[:16]


def attn_profiled_traffic(workload: str):
    path = os.path.join(ROOT, "profiles", f"paged_attn_kernel_{workload}.md")
    if not os.path.exists(path):
        return None
    text = open(path).read()
    m = re.search(r"traffic_bytes_per_launch:\s*(\d+)", text)
    s = re.search(r"source_sha:\s*([0-9a-f]+)", text)
    if not m or not s or s.group(1) != attn_source_sha():
        return None
    return int(m.group(1))


def attn_oracle_sample(w, seed: int, target_s: float, threads: int = 1, nseq_fixed: int = 0):
    """Times the fp64 oracle on whole sequences of the workload (shortest
    first, sequences regenerated on the host) until about target_s seconds
    have been spent, or on the first nseq_fixed sequences spread over
    `threads` threads; returns (seconds, tokens of context processed,
    sequences)."""
    import oracle
    from paper_2412_15803_gb300 import synth
    sh = w.shape
    lens = w.lens(seed)
    P, D = w.page_size, sh.head_dim
    num_pages = int(((lens.astype(np.int64) + P - 1) // P).sum())
    table = synth.page_table(seed, lens, P, num_pages)
    per = sh.n_kv_heads * P * D
    def inputs(b):
        T = int(lens[b])
        n = (T + P - 1) // P
        pages = table[b, :n]
        k = np.stack([synth.sum4_fp16(seed, synth.stream_id(synth.KIND_K, 0, 0), int(p) * per, per) for p in pages])
        v = np.stack([synth.sum4_fp16(seed, synth.stream_id(synth.KIND_V, 0, 0), int(p) * per, per) for p in pages])
        k = k.reshape(n, sh.n_kv_heads, P, D)
        v = v.reshape(n, sh.n_kv_heads, P, D)
        q = synth.sum4_fp16(seed, synth.stream_id(synth.KIND_Q, 0, 0), int(b) * sh.n_q_heads * D, sh.n_q_heads * D)
        return q, k, v, n, T

    def call(a):
        q, k, v, n, T = a
        oracle.paged_attention(q[None, :], k, v, np.arange(n, dtype=np.int32)[None, :], np.array([T], np.int32),
                               1.0 / np.sqrt(D), sh.n_q_heads)

    order = np.argsort(lens, kind="stable")
    if threads > 1 and nseq_fixed:
        # the same sequences, one per thread at a time (the C routine releases the GIL)
        from concurrent.futures import ThreadPoolExecutor
        args = [inputs(b) for b in order[:nseq_fixed]]
        with ThreadPoolExecutor(threads) as ex:
            t0 = time.perf_counter()
            list(ex.map(call, args))
            spent = time.perf_counter() - t0
        return spent, sum(a[4] for a in args), len(args)
    spent, toks, nseq = 0.0, 0, 0
    for b in order:
        a = inputs(b)
        t0 = time.perf_counter()
        call(a)
        spent += time.perf_counter() - t0
        toks += a[4]
        nseq += 1
        if spent >= target_s:
            break
    return spent, toks, nseq


def attn_cpu_line(w, seed: int, target_s: float):
    t, toks, nseq = attn_oracle_sample(w, seed, target_s)
    total_toks = int(w.lens(seed).astype(np.int64).sum())
    est = t * total_toks / max(toks, 1)
    host = host_info()
    line = {"value": w.batch / est, "unit": "sequences/s", "cores": 1, "kind": "oracle",
            "sample": f"{nseq} of the {w.batch} sequences (shortest first, {toks} of {total_toks} context "
                      f"tokens), single-threaded fp64 C oracle, {t:.1f} s, scaled to the whole batch", **host}
    threads = host["nproc"]
    if threads > 1 and nseq >= 2:
        tp, toksp, nseqp = attn_oracle_sample(w, seed, target_s, threads=threads, nseq_fixed=nseq)
        line["all_core"] = {"value": w.batch / (tp * total_toks / max(toksp, 1)), "unit": "sequences/s",
                            "cores": threads,
                            "kind": f"oracle, sequence-parallel: the same fp64 C routine, one sequence per "
                                    f"thread on {threads} threads",
                            "sample": f"the same {nseqp} sequences, {tp:.1f} s, scaled to the whole batch"}
    return line


def attn_config(w, layers: int):
    sh = w.shape
    return {"workload": f"{w.name}: decode attention of one {sh.name}-shaped layer ({sh.n_q_heads} q / "
                        f"{sh.n_kv_heads} kv heads of {sh.head_dim}), batch {w.batch}, context lengths "
                        f"uniform on [{w.len_lo}, {w.len_hi}], pages of {w.page_size} tokens, fp16 cache",
            "batch": w.batch, "page_size": w.page_size,
            "l2": ("inputs larger than L2, no flush" if layers == 1 else
                   f"{layers} distinct layers' caches in rotation (together larger than L2)"),
            "parallelism": "single GPU"}


def run_attn_reference(args, rank, world):
    from paper_2412_15803_gb300.attention import ATTN_WORKLOADS
    if rank != 0:
        return
    w = ATTN_WORKLOADS[args.workload]
    nsteps = args.steps + args.warmup
    step_s = min(10.0, 120.0 / max(nsteps, 1))
    times = []
    total_toks = int(w.lens(0).astype(np.int64).sum())
    for i in range(nsteps):
        t, toks, _ = attn_oracle_sample(w, 0, step_s)
        if i >= args.warmup:
            times.append(t * total_toks / max(toks, 1))
    value = w.batch / statistics.mean(times)
    line = {"metric": ATTN_METRIC, "value": value, "unit": "sequences/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * statistics.mean(times), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded sum4 keys, values and queries; random page tables)", "impl": "reference",
            "config": attn_config(w, 1),
            "cpu_baseline": {"value": value, "unit": "sequences/s", "cores": 1, "kind": "oracle",
                             "sample": f"each step: shortest sequences first for about {step_s:.1f} s of oracle "
                                       "time, scaled to the whole batch", **host_info()},
            "e2e": {"value": value, "unit": "sequences/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_attn(args, rank, world, local):
    import torch
    import torch.distributed as dist
    from paper_2412_15803_gb300 import wq4
    from paper_2412_15803_gb300.attention import ATTN_WORKLOADS, PagedAttentionLayer

    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    w = ATTN_WORKLOADS[args.workload]
    lens = w.lens(0)
    first = PagedAttentionLayer(w.shape, lens, page_size=w.page_size, seed=0, layer=0)
    nlayers = 1
    if first.kv_bytes() < 4 * L2_BYTES:
        nlayers = int(np.ceil(4 * L2_BYTES / first.kv_bytes()))
    layers = [first] + [PagedAttentionLayer(w.shape, lens, page_size=w.page_size, seed=0, layer=l)
                        for l in range(1, nlayers)]
    # one step = launches over the layer caches in turn (at least 8), captured
    # once in a CUDA graph as a decode step would be, so host-side call and
    # graph-launch overheads stay out of the per-launch time
    per_graph = max(nlayers, 8)
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        for L in layers:
            L.run(stream)
        stream.synchronize()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=stream):
            for j in range(per_graph):
                layers[j % nlayers].run(stream)
        for _ in range(max(args.warmup, 3)):
            graph.replay()
    torch.cuda.synchronize()
    if wq4.wq4_device_status(stream) != 0:
        raise RuntimeError("attention flagged an error during warm-up")
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.3)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        for i in range(args.steps):
            starts[i].record(stream)
            graph.replay()
            ends[i].record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clocks = sampler.stop()
    total_ms = starts[0].elapsed_time(ends[-1])
    launch_ms = [s.elapsed_time(e) / per_graph for s, e in zip(starts, ends)]
    if wq4.wq4_device_status(stream) != 0:
        raise RuntimeError("attention flagged an error during the timed region")

    # end to end: queries copied in from pinned host memory, the call, outputs copied back
    L0 = layers[0]
    q_host = L0.q.cpu().pin_memory()
    o_host = torch.empty_like(L0.out, device="cpu").pin_memory()
    e2e_steps = max(10, min(args.steps, 500))
    with torch.cuda.stream(stream):
        t0 = time.perf_counter()
        for i in range(e2e_steps):
            Li = layers[i % nlayers]
            Li.q.copy_(q_host, non_blocking=True)
            Li.run(stream)
            o_host.copy_(Li.out, non_blocking=True)
            stream.synchronize()
        e2e_s = time.perf_counter() - t0
    # a step attends every layer cache once: batch sequences per layer launch
    seq_per_s, e2e_val, total_ms_max = aggregate_replicas(total_ms / per_graph, e2e_s / e2e_steps, w.batch,
                                                          args.steps, "cuda")
    if rank == 0:
        avg_launch_ms = statistics.mean(launch_ms)
        peak, peak_src = measured_peak()
        step_bytes = L0.algorithmic_bytes()
        achieved = step_bytes / (avg_launch_ms * 1e-3) / 1e9
        line = {
            "metric": ATTN_METRIC, "value": seq_per_s, "unit": "sequences/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": total_ms_max / args.steps,
            "launches_per_step": per_graph, "layer_caches": nlayers,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "precision": "fp16 cache and queries, fp32 scores and sums, weights rounded to fp16 for the value product",
            "data": "synthetic (seeded sum4 keys, values and queries; random page tables)",
            "config": attn_config(w, nlayers),
            "hbm_gbs": step_bytes * args.steps / (total_ms_max / 1e3) / 1e9,
            "timing": "CUDA-graph replays of launches_per_step launches over the layer caches in turn; "
                      "ms_per_step and value are per launch",
            "roofline": {"bound": "hbm", "kernel": "paged_attn_kernel", "achieved": achieved, "peak": peak,
                         "peak_source": peak_src, "unit": "GB/s", "frac": achieved / peak,
                         "frac_of_nominal_8tbs": achieved / NOMINAL_HBM_GBS,
                         "traffic": attn_profiled_traffic(args.workload),
                         "algorithmic_bytes_per_launch": step_bytes, "avg_launch_ms": avg_launch_ms},
            "e2e": {"value": e2e_val, "unit": "sequences/s", "h2d_bytes_per_step": L0.q.numel() * 2,
                    "d2h_bytes_per_step": L0.out.numel() * 2},
            "gpu_launches": args.steps * per_graph,
            "clocks": clocks,
        }
        if world == 1 and not args.no_cpu_baseline:
            line["cpu_baseline"] = attn_cpu_line(w, 0, 12.0)
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


# ---------------------------------------------------------------- prefill --

PREFILL_METRIC = "prefill-shaped 4-bit dequant-GEMM TFLOP/s (one layer's four projections over a prompt)"


def prefill_projections(shape):
    """(name, N, K, input width) of one layer's projections."""
    return [(n, N, K, K) for n, N, K, _ in shape.mats(0)]


def run_prefill_reference(args, rank, world):
    import oracle
    from paper_2412_15803_gb300 import synth
    from paper_2412_15803_gb300.model import SHAPES
    if rank != 0:
        return
    shape = SHAPES["3b"]
    M = args.tokens
    flops_step = 2 * M * sum(N * K for _, N, K, _ in prefill_projections(shape))
    times, done = [], 0
    nsteps = args.steps + args.warmup
    step_s = min(10.0, 120.0 / max(nsteps, 1))
    x = {K: synth.activations(7, M, K) for K in {shape.hidden, shape.ffn}}
    for i in range(nsteps):
        t_used, f_done = 0.0, 0
        for name, N, K, _ in prefill_projections(shape):
            rows = max(1, int(8 * step_s / 4))    # a few rows of every projection, all tokens
            W, sc = synth.matrix(0, N, K, 0, 0, 0, rows)
            t0 = time.perf_counter()
            oracle.gemv(W, sc, x[K][: max(1, min(M, 64))])
            t_used += time.perf_counter() - t0
            f_done += 2 * rows * K * max(1, min(M, 64))
            if t_used > step_s:
                break
        if i >= args.warmup:
            times.append(t_used)
            done += f_done
    value = done / sum(times) / 1e12
    line = {"metric": PREFILL_METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * flops_step / (value * 1e12), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded SplitMix64 weights and activations)", "impl": "reference",
            "config": {"workload": f"prefill-3b: QKV, O, gate_up, down of one 3B-shaped layer over {M} tokens"},
            "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": 1, "kind": "oracle",
                             "sample": "a few rows of every projection against up to 64 tokens, single-threaded fp64 C oracle",
                             **host_info()},
            "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def measured_tensor_peak():
    try:
        d = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
        return float(d["bf16_tflops"]), "measured (MEASURED_PEAKS.json bf16_tflops, cuBLAS bf16 burst; fp16 runs at the bf16 rate)"
    except Exception:
        return 1900.0, "fallback"


def run_prefill(args, rank, world, local):
    import torch
    import torch.distributed as dist
    from paper_2412_15803_gb300 import synth, wq4
    from paper_2412_15803_gb300.model import SHAPES, fill_matrix

    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    shape = SHAPES["3b"]
    M = args.tokens
    projs = prefill_projections(shape)
    nlayers = 4   # weights of four layers in rotation: 226 MB, larger than L2
    weights = []
    for l in range(nlayers):
        ws = []
        for i, (name, N, K, _) in enumerate(projs):
            W = torch.empty((N, K // 8), dtype=torch.int32, device="cuda")
            sc = torch.empty((N, K // 32), dtype=torch.int16, device="cuda")
            fill_matrix(W, sc, N, K, 0, l, i)
            ws.append((W, sc))
        weights.append(ws)
    xin = {K: torch.from_numpy(synth.activations(7, M, K).view(np.int16)).cuda() for K in {shape.hidden, shape.ffn}}
    outs = [torch.empty((M, N), dtype=torch.int16, device="cuda") for _, N, _, _ in projs]
    flops_step = 2 * M * sum(N * K for _, N, K, _ in projs)

    def step(l, stream):
        for i, (name, N, K, _) in enumerate(projs):
            W, sc = weights[l][i]
            wq4.wq4_gemm(W, sc, xin[K], outs[i], N, K, M, stream)

    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        step(0, stream)
        stream.synchronize()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=stream):
            for l in range(nlayers):
                step(l, stream)
        for _ in range(max(args.warmup, 3)):
            graph.replay()
    torch.cuda.synchronize()
    if wq4.wq4_device_status(stream) != 0:
        raise RuntimeError("device flag set during warm-up")
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.3)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        for i in range(args.steps):
            starts[i].record(stream)
            graph.replay()
            ends[i].record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clocks = sampler.stop()
    total_ms = starts[0].elapsed_time(ends[-1]) / nlayers
    step_ms = [s.elapsed_time(e) / nlayers for s, e in zip(starts, ends)]
    # end to end: inputs copied in from pinned host memory, outputs copied back
    x_host = {K: v.cpu().pin_memory() for K, v in xin.items()}
    o_host = [torch.empty_like(o, device="cpu").pin_memory() for o in outs]
    e2e_steps = max(3, min(args.steps, 20))
    with torch.cuda.stream(stream):
        t0 = time.perf_counter()
        for i in range(e2e_steps):
            for K, v in xin.items():
                v.copy_(x_host[K], non_blocking=True)
            step(i % nlayers, stream)
            for o, oh in zip(outs, o_host):
                oh.copy_(o, non_blocking=True)
            stream.synchronize()
        e2e_s = (time.perf_counter() - t0) / e2e_steps
    if wq4.wq4_device_status(stream) != 0:
        raise RuntimeError("device flag set during the timed region")
    t = torch.tensor([total_ms, e2e_s], dtype=torch.float64, device="cuda")
    if world > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    job_ms, e2e_step = float(t[0]), float(t[1])
    if rank == 0:
        peak, src = measured_tensor_peak()
        avg = statistics.mean(step_ms)
        achieved = flops_step / (avg * 1e-3) / 1e12
        line = {
            "metric": PREFILL_METRIC, "value": world * flops_step * args.steps / (job_ms * 1e-3) / 1e12,
            "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": job_ms / args.steps, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f16",
            "precision": "int4 codes dequantized to fp16 (one rounding), fp16 activations, fp32 accumulation",
            "data": "synthetic (seeded SplitMix64 weights and activations)",
            "config": {"workload": f"prefill-3b: QKV 5120x3072, O 3072x3072, gate_up 16384x3072, down 3072x8192 "
                                   f"of one 3B-shaped layer over {M} prompt tokens (wq4_gemm, tcgen05)",
                       "tokens": M, "flop_per_step": flops_step,
                       "l2": f"{nlayers} layers' weights in rotation (226 MB, larger than L2)",
                       "parallelism": "single GPU"},
            "prefill_tokens_per_s_per_layer": world * M * args.steps / (job_ms * 1e-3),
            "roofline": {"bound": "tensor", "kernel": "gemm_kernel", "achieved": achieved, "peak": peak,
                         "peak_source": src, "unit": "TFLOP/s", "frac": achieved / peak, "traffic": None,
                         "algorithmic_flop_per_step": flops_step, "avg_step_ms": avg},
            "e2e": {"value": flops_step / e2e_step / 1e12, "unit": "TFLOP/s",
                    "h2d_bytes_per_step": sum(v.numel() * 2 for v in xin.values()),
                    "d2h_bytes_per_step": sum(o.numel() * 2 for o in outs)},
            "gpu_launches": args.steps * nlayers * len(projs),
            "clocks": clocks,
        }
        if world == 1 and not args.no_cpu_baseline:
            import oracle
            W, sc = synth.matrix(0, 16, shape.hidden)
            xs = synth.activations(7, 64, shape.hidden)
            t0 = time.perf_counter()
            n = 0
            while time.perf_counter() - t0 < 10.0:
                oracle.gemv(W, sc, xs)
                n += 1
            dt = time.perf_counter() - t0
            host = host_info()
            pool = RowPool(host["nproc"])
            rows = 16 * pool.threads
            Wp, scp = synth.matrix(0, rows, shape.hidden)
            t0 = time.perf_counter()
            npar = 0
            while time.perf_counter() - t0 < 5.0:
                pool.gemv(Wp, scp, xs)
                npar += 1
            dtp = time.perf_counter() - t0
            pool.close()
            line["cpu_baseline"] = {"value": n * 2 * 16 * shape.hidden * 64 / dt / 1e12, "unit": "TFLOP/s", "cores": 1,
                                    "kind": "oracle",
                                    "sample": f"16 rows x {shape.hidden} x 64 tokens repeated for {dt:.1f} s, "
                                              "single-threaded fp64 C oracle", **host,
                                    "all_core": all_core_line(npar * 2 * rows * shape.hidden * 64 / dtp / 1e12,
                                                              "TFLOP/s", pool.threads,
                                                              f"{rows} rows x {shape.hidden} x 64 tokens repeated "
                                                              f"for {dtp:.1f} s")}
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def main():
    args = parse()
    rank, world, local = dist_env()
    if args.workload.startswith("gemv"):
        (run_gemv_reference(args, rank, world) if args.impl == "reference" else run_gemv(args, rank, world, local))
        return
    if args.workload.startswith("prefill"):
        (run_prefill_reference(args, rank, world) if args.impl == "reference" else run_prefill(args, rank, world, local))
        return
    attn = args.workload.startswith("attn")
    if args.impl == "reference":
        (run_attn_reference if attn else run_reference)(args, rank, world)
    else:
        (run_attn if attn else run_ours)(args, rank, world, local)


if __name__ == "__main__":
    main()
