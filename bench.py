"""Benchmark: batched paged-KV decode attention on one GB300 (per rank).

Headline workload: the mixed heavy-tailed rollout batch -- 512 trajectories,
context lengths lognormal (median 4096, sigma 1) clipped to [512, 131072],
64 query / 8 KV heads, head dim 128, 16-token pages in a shuffled pool (about
14 GB of bf16 KV, far larger than L2).  A step is one decode_attention call
over the whole batch for one layer: the planner launch plus the attention
launch (the split-KV merge runs inside the attention kernel).

Printed: one JSON line with the achieved HBM GB/s of algorithmic bytes
(K and V of every context token once per KV head, plus q, out, lse, the
block-table entries used and context_lens), decode steps/s, the attention
kernel's roofline fraction, an end-to-end number through the C ABI with
host buffers, the fp64 CPU oracle timed on a bounded sample, SM clocks
during the timed region and, as a secondary measurement, prefix staging.

``--impl reference`` times the oracle (the library's fp64 CPU reference) on
the same workload and prints the same metric.
Multi-GPU (torchrun): each rank runs its own batch (weak scaling, no
collective on the data path); rank 0 prints the whole-job numbers.
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
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import paper_2609_36899_gb300 as cadkv  # noqa: E402
from paper_2609_36899_gb300 import build as pkg_build  # noqa: E402
from paper_2609_36899_gb300.workloads import (DECODE_WORKLOADS, PREFILL, STAGING,  # noqa: E402
                                              bf16_bits, fill_layer_pool, landscape_workload,
                                              COMPOSITIONS, composition_workload,
                                              make_decode_batch, make_prefill_job,
                                              make_staging_job)

METRIC = "decode-attention achieved HBM GB/s (% of 8 TB/s) and decode steps/s per batch"
NOMINAL_HBM_GBS = 8000.0
PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")
FALLBACK_HBM_GBS = 6800.0
PROFILE_SUMMARY = os.path.join(ROOT, "profiles", "decode_attention_kernel_mixed_b512_dram.md")
STAGE_PROFILE_SUMMARY = os.path.join(ROOT, "profiles", "stage_copy_kernel_staging_8traj_1layer.md")
KERNEL_SOURCE = os.path.join(ROOT, "paper_2609_36899_gb300", "csrc", "decode_attention.cu")
STAGE_SOURCE = os.path.join(ROOT, "paper_2609_36899_gb300", "csrc", "prefix_stage.cu")


# ------------------------------------------------------------------ helpers

def hbm_peak():
    try:
        with open(PEAKS_FILE) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def source_hash(path):
    with open(path, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


def profiled_traffic(summary_path, source_path, key="dram_bytes_per_launch"):
    """A DRAM-traffic figure (``key``) from a committed ncu summary, or None
    when the summary is missing or was taken on a different kernel source."""
    try:
        text = open(summary_path).read()
    except OSError:
        return None
    m = re.search(r"kernel_source_sha256_16:\s*([0-9a-f]{16})", text)
    t = re.search(re.escape(key) + r":\s*([0-9.eE+]+)", text)
    if not m or not t or m.group(1) != source_hash(source_path):
        return None
    return float(t.group(1))


class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons every 200 ms."""
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device):
        self.proc = None
        try:
            self.gpu_id = "GPU-" + str(torch.cuda.get_device_properties(device).uuid)
        except Exception:
            self.gpu_id = str(device.index or 0)

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu_id}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, ValueError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, sm_max, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                sm_max.append(float(parts[1]))
            except ValueError:
                continue
            for name, val in zip(names, parts[4:8]):
                if val.lower() == "active":
                    reasons.add(name)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(sm_max),
                "reasons": sorted(reasons), "samples": len(sm)}


def decode_bytes(lens, hq, hkv, d):
    """Algorithmic bytes of one decode step (see module docstring)."""
    lens = np.asarray(lens, dtype=np.int64)
    b = len(lens)
    pages = int((-(-lens // 16)).sum())
    kv = 4 * hkv * d * int(lens.sum())
    qo = 2 * (2 * b * hq * d)
    return kv + qo + 4 * b * hq + 4 * pages + 4 * b


def dist_setup(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        if torch.cuda.is_available():
            torch.cuda.set_device(local)
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    elif torch.cuda.is_available():
        torch.cuda.set_device(0)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64,
                     device="cuda" if dist.get_backend() == "nccl" else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64,
                     device="cuda" if dist.get_backend() == "nccl" else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


# ------------------------------------------------------------------ CPU oracle leg

class OracleSample:
    """A bounded sample of a batch's trajectories, copied to the host once, on
    which the fp64 oracle is timed.

    Trajectories are taken in a seeded shuffled order until the estimated
    oracle time (from a one-trajectory pilot) reaches ``target_s``.
    """

    def __init__(self, batch, target_s: float, threads: int | None = None):
        import oracle
        oracle.build()
        self.orc = oracle.default()
        self.threads = threads or len(os.sched_getaffinity(0))
        w = batch.workload
        lens = batch.context_lens
        order = np.random.Generator(np.random.PCG64(w.seed + 99)).permutation(len(lens))
        pilot = self._inputs(batch, [int(order[0])])
        t = self._time(pilot)
        budget_tokens = max(int(lens[order[0]]), 1) / max(t, 1e-6) * target_s
        chosen, tokens = [], 0
        for b in order:
            chosen.append(int(b))
            tokens += int(lens[b])
            if tokens >= budget_tokens:
                break
        self.inputs = self._inputs(batch, chosen)
        sel = lens[np.array(chosen)]
        self.nbytes = decode_bytes(sel, w.num_q_heads, w.num_kv_heads, w.head_dim)
        self.desc = (f"{len(chosen)} of {len(lens)} trajectories of the same batch "
                     f"({int(sel.sum())} context tokens, all {w.num_q_heads} query heads), "
                     f"fp64 oracle, OpenMP {self.threads} threads")

    @staticmethod
    def _inputs(batch, chosen):
        lens = batch.context_lens[np.array(chosen)]
        pages = -(-lens.astype(np.int64) // 16)
        phys = np.concatenate([batch.block_table[b, :p] for b, p in zip(chosen, pages)])
        idx = torch.from_numpy(phys.astype(np.int64)).to(batch.k_pages.device)
        k = bf16_bits(batch.k_pages.index_select(0, idx))
        v = bf16_bits(batch.v_pages.index_select(0, idx))
        q = bf16_bits(batch.q[torch.as_tensor(chosen, device=batch.q.device)])
        table = np.full((len(chosen), max(int(pages.max()), 1)), -1, dtype=np.int32)
        pos = 0
        for i, p in enumerate(pages):
            table[i, :p] = np.arange(pos, pos + p)
            pos += p
        return q, k, v, table, lens

    def _time(self, inputs):
        t0 = time.perf_counter()
        self.orc.decode_attention(*inputs, num_threads=self.threads)
        return time.perf_counter() - t0

    def run(self) -> float:
        """Seconds for one oracle evaluation of the sample."""
        return self._time(self.inputs)


def oracle_staging_baseline(job, k_layers, v_layers, target_s=4.0):
    """The oracle's prefix gather (C, OpenMP over the host cores) on a bounded
    sample of the job's trajectories, one layer: GB/s read + write."""
    import oracle
    oracle.build()
    orc = oracle.default()
    threads = len(os.sched_getaffinity(0))
    lens = job.context_lens
    order = np.random.Generator(np.random.PCG64(STAGING.seed + 99)).permutation(len(lens))

    def sample(chosen):
        sel = lens[np.array(chosen)]
        pages = -(-sel.astype(np.int64) // 16)
        phys = np.concatenate([job.block_table[b, :pg] for b, pg in zip(chosen, pages)])
        idx = torch.from_numpy(phys.astype(np.int64)).to(k_layers[0].device)
        kp = bf16_bits(k_layers[0].index_select(0, idx))[None]
        vp = bf16_bits(v_layers[0].index_select(0, idx))[None]
        table = np.full((len(chosen), int(pages.max())), -1, dtype=np.int32)
        pos = 0
        for i, pg in enumerate(pages):
            table[i, :pg] = np.arange(pos, pos + pg)
            pos += pg
        return kp, vp, table, sel

    def timed(inp):
        t0 = time.perf_counter()
        orc.prefix_stage(inp[0], inp[1], inp[2], inp[3], 0, 1, num_threads=threads)
        return time.perf_counter() - t0

    pilot = sample([int(order[0])])
    per_token = timed(pilot) / max(int(lens[order[0]]), 1)
    chosen, tokens = [], 0
    for b in order:
        chosen.append(int(b))
        tokens += int(lens[b])
        if tokens * per_token >= target_s:
            break
    inp = sample(chosen)
    secs = timed(inp)
    nbytes = 2 * 2 * int(inp[3].sum()) * 8 * 128 * 2  # read + write, K and V, bytes
    return {"value": round(nbytes / secs / 1e9, 3), "unit": "GB/s", "cores": threads,
            "kind": "oracle", "seconds": round(secs, 2),
            "sample": f"{len(chosen)} of {len(lens)} trajectories ({tokens} tokens), 1 layer, "
                      f"C oracle gather, OpenMP {threads} threads"}


def oracle_prefill_baseline(b, offs, q, w, target_s=4.0):
    """The fp64 oracle (C, OpenMP over the host cores) on the last rows of
    trajectory 0's chunk, every query head: TFLOP/s of algorithmic causal flops."""
    import oracle
    oracle.build()
    orc = oracle.default()
    threads = len(os.sched_getaffinity(0))
    n = int(b.context_lens[0])
    npg = -(-n // 16)
    idx = torch.from_numpy(b.block_table[0, :npg].astype(np.int64)).to(b.k_pages.device)
    kp = bf16_bits(b.k_pages.index_select(0, idx))
    vp = bf16_bits(b.v_pages.index_select(0, idx))
    table = np.arange(npg, dtype=np.int32)[None]
    qb = bf16_bits(q[:w.chunk])

    def run(rows):
        sub = np.ascontiguousarray(qb[w.chunk - rows:])
        t0 = time.perf_counter()
        orc.prefill_attention(sub, np.array([0, rows], dtype=np.int64), kp, vp, table,
                              np.array([n], dtype=np.int32), num_threads=threads)
        return time.perf_counter() - t0

    rows = max(1, min(w.chunk, int(target_s / max(run(4) / 4, 1e-9))))
    secs = run(rows)
    pos = np.arange(n - rows, n, dtype=np.float64)
    flops = w.num_q_heads * float((4.0 * w.head_dim * (pos + 1)).sum())
    return {"value": round(flops / secs / 1e12, 6), "unit": "TFLOP/s", "cores": threads,
            "kind": "oracle", "seconds": round(secs, 2),
            "sample": f"last {rows} of the {w.chunk} query tokens of trajectory 0 "
                      f"(context {n}), all {w.num_q_heads} query heads, fp64 oracle, "
                      f"OpenMP {threads} threads"}


# ------------------------------------------------------------------ GPU legs

def time_decode(tensors, steps, warmup, stream):
    q, k, v, bt, cl, out, lse, ws = tensors
    for _ in range(warmup):
        cadkv.decode_attention_plan(q, k, v, bt, cl, out, lse, ws, stream=stream)
        cadkv.decode_attention_run(q, k, v, bt, cl, out, lse, ws, stream=stream)
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True),
           torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    return ev


def run_decode_loop(tensors, ev, stream):
    q, k, v, bt, cl, out, lse, ws = tensors
    for e0, e1, e2 in ev:
        e0.record(stream)
        cadkv.decode_attention_plan(q, k, v, bt, cl, out, lse, ws, stream=stream)
        e1.record(stream)
        cadkv.decode_attention_run(q, k, v, bt, cl, out, lse, ws, stream=stream)
        e2.record(stream)


def time_append_step(batch, tensors, steps, warmup, stream):
    """The whole decode step of one layer, decode_attention_append: write the new
    token's K/V for every trajectory, then attend (2 launches)."""
    q, k, v, bt, cl, out, lse, ws = tensors
    w = batch.workload
    g = torch.Generator(device=q.device).manual_seed(w.seed + 7)
    k_new = torch.randn((q.shape[0], w.num_kv_heads, w.head_dim), generator=g,
                        device=q.device).to(torch.bfloat16)
    v_new = torch.randn_like(k_new, dtype=torch.float32).to(torch.bfloat16)
    for _ in range(warmup):
        cadkv.decode_attention_append(q, k_new, v_new, k, v, bt, cl, out=out, lse=lse,
                                      workspace=ws, stream=stream)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(steps):
        cadkv.decode_attention_append(q, k_new, v_new, k, v, bt, cl, out=out, lse=lse,
                                      workspace=ws, stream=stream)
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / steps
    nbytes = decode_bytes(batch.context_lens, w.num_q_heads, w.num_kv_heads, w.head_dim)
    nbytes += 2 * 2 * k_new.numel() * 2          # read k_new, v_new; write them to the pool
    return {"gbps": round(nbytes / (ms * 1e-3) / 1e9, 1), "ms_per_step": round(ms, 4),
            "steps_per_s": round(1e3 / ms, 1), "launches_per_step": 2,
            "status": cadkv.decode_attention_status(ws)}


def e2e_loop(batch, tensors, steps, warmup, stream):
    """decode_attention through the C ABI with host inputs and outputs: every
    step uploads q, block_table and context_lens from pinned host memory, runs
    the step and downloads out and lse to pinned host memory.  As in a serving
    loop, transfers overlap compute: the device inputs are double-buffered,
    step i + 1's upload runs on a copy stream while step i computes, and step
    i's download follows it on the copy stream (events order the three)."""
    q, k, v, bt, cl, out, lse, ws = tensors
    device = q.device
    hq = batch.q.cpu().pin_memory()
    hbt = torch.from_numpy(batch.block_table).pin_memory()
    hcl = torch.from_numpy(batch.context_lens).pin_memory()
    hout = torch.empty(out.shape, dtype=out.dtype).pin_memory()
    hlse = torch.empty(lse.shape, dtype=lse.dtype).pin_memory()
    bufs = [(q, bt, cl, out, lse),
            (torch.empty_like(q), torch.empty_like(bt), torch.empty_like(cl),
             torch.empty_like(out), torch.empty_like(lse))]
    copy = torch.cuda.Stream(device)
    uploaded = [torch.cuda.Event() for _ in range(2)]
    computed = [torch.cuda.Event() for _ in range(2)]

    def upload(i):
        dq, dbt, dcl = bufs[i % 2][:3]
        with torch.cuda.stream(copy):
            if i >= 2:  # buffer reuse: step i - 2 must be done with it
                copy.wait_event(computed[i % 2])
            dq.copy_(hq, non_blocking=True)
            dbt.copy_(hbt, non_blocking=True)
            dcl.copy_(hcl, non_blocking=True)
            uploaded[i % 2].record(copy)

    def run(n):
        upload(0)
        for i in range(n):
            dq, dbt, dcl, dout, dlse = bufs[i % 2]
            stream.wait_event(uploaded[i % 2])
            cadkv.decode_attention(dq, k, v, dbt, dcl, out=dout, lse=dlse, workspace=ws,
                                   stream=stream)
            computed[i % 2].record(stream)
            if i + 1 < n:
                upload(i + 1)
            with torch.cuda.stream(copy):
                copy.wait_event(computed[i % 2])
                hout.copy_(dout, non_blocking=True)
                hlse.copy_(dlse, non_blocking=True)
        torch.cuda.synchronize(device)

    run(warmup)
    t0 = time.perf_counter()
    run(steps)
    secs = (time.perf_counter() - t0) / steps
    h2d = hq.numel() * 2 + hbt.numel() * 4 + hcl.numel() * 4
    d2h = hout.numel() * 2 + hlse.numel() * 4
    return secs, h2d, d2h


def staging_chunk_layers(pool_layer_bytes, rows_layer_bytes, free_bytes, total_layers=48):
    """Layers per chunk of the staging job: the largest divisor of the layer
    count among 12, 8, 6, 4, 3, 2, 1 whose K/V pool and staged rows fit in 90 %
    of the free device memory."""
    for lc in (12, 8, 6, 4, 3, 2, 1):
        if total_layers % lc == 0 and lc * (pool_layer_bytes + rows_layer_bytes) <= 0.9 * free_bytes:
            return lc
    raise RuntimeError("one layer of the staging job does not fit in device memory")


def bench_staging(device, chunk_layers=None, batch=None, cpu_baseline=False):
    """The whole prefix-staging job: all 48 layers of the staging workload's
    trajectories (all 64, or the first ``batch`` of the same draw).  The job's
    ~464 GB of K/V does not fit in HBM next to its destination, so it runs in
    chunks of ``chunk_layers`` layers (default: the largest that fits): each
    chunk's pool is filled from the per-layer seeds (untimed), staged by one
    kv_prefix_stage call (timed), then loaded back by one kv_prefix_load call
    (timed; the values written equal those already there).  The job time is the
    sum of the chunks' staging times.  One trajectory per chunk is checked bit
    for bit against the pool; the -m gpu tests compare every chunk of the job
    with the oracle's gather."""
    job = make_staging_job(STAGING, batch=batch)
    w = STAGING
    lens = job.context_lens
    hkv, d, total_layers = w.num_kv_heads, w.head_dim, w.num_layers
    page_elems = hkv * 16 * d
    pool_layer_bytes = 2 * job.num_pages * page_elems * 2
    rows_layer = cadkv.staged_size(lens, 0, 1, hkv, d)            # elements per layer
    torch.cuda.empty_cache()
    free, _ = torch.cuda.mem_get_info(device)
    lc = chunk_layers or staging_chunk_layers(pool_layer_bytes, rows_layer * 2, free, total_layers)
    if total_layers % lc:
        raise ValueError(f"{lc} layers per chunk do not divide {total_layers}")
    k_layers = [torch.empty((job.num_pages, hkv, 16, d), dtype=torch.bfloat16, device=device)
                for _ in range(lc)]
    v_layers = [torch.empty_like(k_layers[0]) for _ in range(lc)]
    pool = cadkv.KVPool(k_layers, v_layers)
    size = rows_layer * lc
    dst = torch.empty(size, dtype=torch.bfloat16, device=device)
    bt = torch.from_numpy(job.block_table).to(device)
    cl = torch.from_numpy(lens).to(device)
    ws = torch.empty(cadkv.kv_prefix_stage_workspace_size(len(lens)), dtype=torch.uint8,
                     device=device)
    stream = torch.cuda.current_stream(device)
    row = lc * 2 * hkv * d
    starts = np.concatenate([[0], np.cumsum(lens.astype(np.int64) * row)])
    stage_ms, load_ms, statuses, spot = [], [], [], []
    for c in range(total_layers // lc):
        for i in range(lc):
            fill_layer_pool(k_layers[i], v_layers[i], w.seed, c * lc + i)
        if c == 0:   # warm-up calls (first touch of dst, library set-up)
            for _ in range(2):
                cadkv.kv_prefix_stage(pool, bt, cl, 0, lc, dst, workspace=ws, stream=stream)
        torch.cuda.synchronize()
        e = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
        e[0].record(stream)
        cadkv.kv_prefix_stage(pool, bt, cl, 0, lc, dst, workspace=ws, stream=stream)
        e[1].record(stream)
        cadkv.kv_prefix_load(pool, bt, cl, 0, lc, dst, workspace=ws, stream=stream)
        e[2].record(stream)
        torch.cuda.synchronize()
        stage_ms.append(e[0].elapsed_time(e[1]))
        load_ms.append(e[1].elapsed_time(e[2]))
        statuses.append(cadkv.kv_prefix_stage_status(ws))
        # spot check: one trajectory (a different one per chunk) against the pool
        b = c % len(lens)
        n = int(lens[b])
        p = -(-n // 16)
        got = dst[int(starts[b]):int(starts[b + 1])].view(lc, 2, hkv, n, d)
        phys = bt[b, :p].long()
        ok = True
        for i in range(lc):
            for kv, src in ((0, k_layers[i]), (1, v_layers[i])):
                rows = src.index_select(0, phys).permute(1, 0, 2, 3).reshape(hkv, p * 16, d)
                ok &= bool(torch.equal(rows[:, :n].view(torch.int16), got[i, kv].view(torch.int16)))
        spot.append(ok)
    moved = 2 * size * 2                       # read + write bytes per chunk call
    total_moved = moved * len(stage_ms)
    total_ms = sum(stage_ms)
    peak, kind = hbm_peak()
    gbs = total_moved / (total_ms * 1e-3) / 1e9
    load_gbs = total_moved / (sum(load_ms) * 1e-3) / 1e9
    traffic_ratio = profiled_traffic(STAGE_PROFILE_SUMMARY, STAGE_SOURCE,
                                     key="dram_bytes_per_staged_byte")
    res = {"workload": f"{STAGING.name}: {len(lens)} trajectories x {total_layers} layers "
                       f"({int(lens.sum())} tokens, {hkv} KV heads, D={d}), in "
                       f"{len(stage_ms)} chunks of {lc} layers (pool refilled per chunk)",
           "layers": total_layers, "chunk_layers": lc, "chunks": len(stage_ms),
           "gbps_read_plus_write": round(gbs, 1), "ms_total": round(total_ms, 3),
           "ms_per_chunk": [round(x, 3) for x in stage_ms],
           "bytes_total": total_moved, "bytes_per_chunk": moved, "launches_per_chunk": 2,
           "status": min(statuses) if statuses else 0,
           "bit_exact_spot_check_vs_pool": all(spot),
           "frac_of_copy_peak": round(gbs / peak, 4),
           "load": {"gbps_read_plus_write": round(load_gbs, 1),
                    "ms_total": round(sum(load_ms), 3),
                    "frac_of_copy_peak": round(load_gbs / peak, 4)},
           "roofline": {"bound": "hbm", "achieved": round(gbs, 1), "peak": peak,
                        "unit": "GB/s", "frac": round(gbs / peak, 4),
                        "peak_kind": kind, "kernel": "stage_copy_kernel<128>",
                        "traffic": (None if traffic_ratio is None
                                    else round(traffic_ratio * size * 2))}}
    if cpu_baseline:
        res["cpu_baseline"] = oracle_staging_baseline(job, k_layers, v_layers)
    del dst, k_layers, v_layers, pool
    torch.cuda.empty_cache()
    return res


def bench_host_staging(device, reps, layers=2, batch=8):
    """Prefix staging to and from page-locked host memory: the copy kernel reads
    the pool and writes the rows straight over the CPU-GPU link (and the inverse
    for the load).  The link's own figure is a cudaMemcpyAsync of the same bytes
    between a device buffer and the same pinned buffer."""
    job = make_staging_job(STAGING, batch=batch)
    k_layers = [torch.empty((job.num_pages, 8, 16, 128), dtype=torch.bfloat16, device=device)
                for _ in range(layers)]
    v_layers = [torch.empty_like(k_layers[0]) for _ in range(layers)]
    for l in range(layers):
        fill_layer_pool(k_layers[l], v_layers[l], STAGING.seed, l)
    pool = cadkv.KVPool(k_layers, v_layers)
    lens = job.context_lens
    size = cadkv.staged_size(lens, 0, layers, 8, 128)
    host = torch.empty(size, dtype=torch.bfloat16, pin_memory=True)
    dev = torch.empty(size, dtype=torch.bfloat16, device=device)
    bt = torch.from_numpy(job.block_table).to(device)
    cl = torch.from_numpy(lens).to(device)
    ws = torch.empty(cadkv.kv_prefix_stage_workspace_size(len(lens)), dtype=torch.uint8,
                     device=device)
    stream = torch.cuda.current_stream(device)

    def timed(fn):
        for _ in range(2):
            fn()
        torch.cuda.synchronize()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(reps)]
        for e0, e1 in ev:
            e0.record(stream)
            fn()
            e1.record(stream)
        torch.cuda.synchronize()
        return statistics.mean(e0.elapsed_time(e1) for e0, e1 in ev)

    to_host_ms = timed(lambda: cadkv.kv_prefix_stage(pool, bt, cl, 0, layers, host,
                                                     workspace=ws, stream=stream))
    to_host_status = cadkv.kv_prefix_stage_status(ws)
    cadkv.kv_prefix_stage(pool, bt, cl, 0, layers, dev, workspace=ws, stream=stream)
    torch.cuda.synchronize()
    exact = bool(torch.equal(host.to(device, non_blocking=False).view(torch.int16),
                             dev.view(torch.int16)))
    from_host_ms = timed(lambda: cadkv.kv_prefix_load(pool, bt, cl, 0, layers, host,
                                                      workspace=ws, stream=stream))
    from_host_status = cadkv.kv_prefix_stage_status(ws)
    d2h_ms = timed(lambda: host.copy_(dev, non_blocking=True))
    h2d_ms = timed(lambda: dev.copy_(host, non_blocking=True))
    nbytes = size * 2

    def gbs(ms):
        return round(nbytes / (ms * 1e-3) / 1e9, 1)

    res = {"workload": f"{STAGING.name}: first {len(lens)} trajectories, {layers} of 48 layers, "
                       "rows in page-locked host memory",
           "bytes_over_link_per_call": nbytes,
           "to_host": {"gbps": gbs(to_host_ms), "ms_per_call": round(to_host_ms, 3),
                       "status": to_host_status, "bit_exact_vs_device_staging": exact,
                       "frac_of_memcpy_d2h": round(d2h_ms / to_host_ms, 4)},
           "from_host": {"gbps": gbs(from_host_ms), "ms_per_call": round(from_host_ms, 3),
                         "status": from_host_status,
                         "frac_of_memcpy_h2d": round(h2d_ms / from_host_ms, 4)},
           "link_reference": {"memcpy_d2h_gbps": gbs(d2h_ms), "memcpy_h2d_gbps": gbs(h2d_ms),
                              "note": "cudaMemcpyAsync of the same bytes, contiguous, no gather"}}
    del host, dev, k_layers, v_layers, pool
    torch.cuda.empty_cache()
    return res


def read_probe(buf, reps=10):
    """Pure-read bandwidth (GB/s) of ``buf`` with the library's read probe."""
    sink = torch.zeros(1, dtype=torch.int64, device=buf.device)
    stream = torch.cuda.current_stream(buf.device)
    for _ in range(3):
        cadkv.cadkv_hbm_read_probe(buf, sink, stream=stream)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(reps):
        cadkv.cadkv_hbm_read_probe(buf, sink, stream=stream)
    e1.record(stream)
    torch.cuda.synchronize()
    return buf.numel() * buf.element_size() * reps / (e0.elapsed_time(e1) * 1e-3) / 1e9


L2_BYTES = 129 << 20   # GB300 L2 (per GPU)
LAYERS_PER_ITERATION = 36  # Qwen3-8B, the paper's main rollout model


def _decode_cell(w, device, steps, warmup):
    """Back-to-back decode steps of one workload: GB/s, time and steps/s, from
    the better of two timed runs of ``steps`` steps (both are reported).

    A decode step is one layer's attention.  As in a model's layer loop, step i
    reads layer i mod L of L layers of KV pages (same lengths and tables, other
    values), with L chosen so that the L layers together exceed three times the
    L2, so that no step finds its pages in L2 (L = 1 when one layer already
    does).  ``same_layer`` repeats layer 0 instead, the way the cell was timed
    before; small cells then stream from L2.  ``plan_per_iteration`` plans once
    per LAYERS_PER_ITERATION steps (one decode iteration of a model of that
    depth: the plan depends only on the lengths) and runs each step on it.

    Eager: one call per step from Python (a DecodeStep, the binding's prepared
    form of decode_attention), so a step can be no shorter than the host's time
    to issue it (host_us_per_call).  Graph: the same calls captured once in a
    CUDA graph and replayed, as a serving engine issues its decode steps: the
    device time."""
    batch = make_decode_batch(w, device=device)
    tensors = _tensors(batch, device)
    stream = torch.cuda.Stream(device)
    q, k, v, bt, cl, out, lse, ws = tensors
    layer_bytes = 2 * k.numel() * k.element_size()
    n_layers = max(1, min(32, -(-3 * L2_BYTES // layer_bytes)))
    layers = [(k, v)]
    for l in range(1, n_layers):
        g = torch.Generator(device=device).manual_seed(w.seed * 1000 + l)
        layers.append(tuple(torch.randn(k.shape, generator=g, device=device,
                                        dtype=torch.float32).to(torch.bfloat16)
                            for _ in range(2)))

    # one prepared call per layer: the tensors are checked and marshalled once
    calls = [cadkv.DecodeStep(q, kl, vl, bt, cl, out, lse, ws, stream=stream)
             for kl, vl in layers]
    plan = cadkv.DecodeStep(q, k, v, bt, cl, out, lse, ws, stream=stream, launch="plan")
    runs_only = [cadkv.DecodeStep(q, kl, vl, bt, cl, out, lse, ws, stream=stream, launch="run")
                 for kl, vl in layers]

    def step(l):
        calls[l]()

    def timed(fn, reps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        fn()
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / reps

    def rotating():
        for i in range(steps):   # back to back: the planner/attention overlap is kept
            step(i % n_layers)

    def same_layer():
        for _ in range(steps):
            step(0)

    def planned_per_iteration():
        # a decode iteration of a model with LAYERS_PER_ITERATION layers plans
        # once and runs every layer on that plan
        for i in range(steps):
            if i % LAYERS_PER_ITERATION == 0:
                plan()
            runs_only[i % n_layers]()

    res = {}
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        for _ in range(warmup):
            step(0)
        torch.cuda.synchronize()
        for name, loop in (("rotating", rotating), ("same_layer", same_layer),
                           ("plan_per_iteration", planned_per_iteration)):
            # a cell timed right after much larger ones was sometimes slow once
            runs = [timed(loop, steps) for _ in range(2)]
            t0 = time.perf_counter()
            loop()
            host_us = (time.perf_counter() - t0) / steps * 1e6
            torch.cuda.synchronize()
            graph = torch.cuda.CUDAGraph()
            with torch.cuda.graph(graph, stream=stream):
                loop()
            graph.replay()
            torch.cuda.synchronize()
            graph_runs = [timed(graph.replay, steps) for _ in range(2)]
            del graph
            res[name] = (runs, graph_runs, host_us)
    nbytes = decode_bytes(batch.context_lens, w.num_q_heads, w.num_kv_heads, w.head_dim)

    def summary(runs, graph_runs, host_us):
        ms, gms = min(runs), min(graph_runs)
        return {"gbps": round(nbytes / (ms * 1e-3) / 1e9, 1), "ms_per_step": round(ms, 4),
                "ms_per_step_runs": [round(r, 4) for r in runs],
                "steps_per_s": round(1e3 / ms, 1),
                "host_us_per_call": round(host_us, 2),
                "graph": {"gbps": round(nbytes / (gms * 1e-3) / 1e9, 1),
                          "ms_per_step": round(gms, 4),
                          "ms_per_step_runs": [round(r, 4) for r in graph_runs]}}

    cell = summary(*res["rotating"])
    cell["tokens_per_s_per_layer"] = round(w.batch * 1e3 / cell["ms_per_step"], 1)
    cell["layers_rotated"] = n_layers
    cell["same_layer"] = summary(*res["same_layer"])
    cell["plan_per_iteration"] = summary(*res["plan_per_iteration"])
    cell["max_context"] = int(batch.context_lens.max())
    cell["status"] = cadkv.decode_attention_status(ws, stream)
    del calls, plan, runs_only, layers, batch, tensors, q, k, v, bt, cl, out, lse, ws
    torch.cuda.empty_cache()
    return cell


def bench_landscape(device, steps, warmup, batches=(8, 32, 128, 512, 2048),
                    means=(256, 1024, 4096, 16384, 65536), max_tokens=8 << 20):
    """Decode GB/s and steps/s over (B, mean context), 32/8 heads, D = 128."""
    cells = []
    for b in batches:
        for c in means:
            if b * c > max_tokens:
                continue
            cells.append({"batch": b, "mean_context": c,
                          **_decode_cell(landscape_workload(b, c), device, steps, warmup)})
    return cells


def bench_composition(device, steps, warmup, batches=(32, 128), mean=4096):
    """Decode GB/s at a fixed batch size and mean context for five within-batch
    length compositions (equal ... one trajectory holding half the tokens)."""
    return [{"batch": b, "mean_context": mean, "composition": comp,
             **_decode_cell(composition_workload(b, mean, comp), device, steps, warmup)}
            for b in batches for comp in COMPOSITIONS]


def bench_prefill(device, steps, warmup, cpu_baseline=False):
    """Chunked re-prefill: each of 8 trajectories recomputes attention for its
    last 512 tokens over a 16,384-token paged KV (32/8 heads, D=128)."""
    w = PREFILL
    batch, context, chunk, hq, hkv = w.batch, w.context, w.chunk, w.num_q_heads, w.num_kv_heads
    b, offs, q = make_prefill_job(w, device)
    bt = torch.from_numpy(b.block_table).to(device)
    cl = torch.from_numpy(b.context_lens).to(device)
    out = torch.empty_like(q)
    lse = torch.empty((batch * chunk, hq), dtype=torch.float32, device=device)
    ws = torch.empty(max(int(cadkv.library().prefill_attention_workspace_size(batch)), 1),
                     dtype=torch.uint8, device=device)
    stream = torch.cuda.current_stream(device)
    for _ in range(warmup):
        cadkv.prefill_attention(q, offs, b.k_pages, b.v_pages, bt, cl, out=out, lse=lse,
                                workspace=ws, stream=stream)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(steps):
        cadkv.prefill_attention(q, offs, b.k_pages, b.v_pages, bt, cl, out=out, lse=lse,
                                workspace=ws, stream=stream)
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / steps
    # algorithmic flops: each (row, head) at position p does 2 D (p + 1) for QK^T and for PV
    pos = np.arange(context - chunk, context, dtype=np.float64)
    flops = batch * hq * float((4.0 * 128 * (pos + 1)).sum())
    try:
        peak = float(json.load(open(PEAKS_FILE))["bf16_tflops"])
        kind = "measured"
    except Exception:
        peak, kind = 1900.0, "fallback"
    tflops = flops / (ms * 1e-3) / 1e12
    res = {"workload": f"chunked prefill: {batch} trajectories x last {chunk} of {context} "
                       f"tokens, {hq}/{hkv} heads, D=128, causal",
           "ms_per_call": round(ms, 4), "tflops": round(tflops, 1),
           "status": cadkv.prefill_attention_status(ws), "launches_per_call": 2,
           "roofline": {"bound": "tensor", "achieved": round(tflops, 1), "peak": peak,
                        "unit": "TFLOP/s", "frac": round(tflops / peak, 4), "peak_kind": kind}}
    if cpu_baseline:
        res["cpu_baseline"] = oracle_prefill_baseline(b, offs, q, w)
    del b, q, out
    torch.cuda.empty_cache()
    return res


def bench_config(name, device, steps, warmup):
    w = DECODE_WORKLOADS[name]
    batch = make_decode_batch(w, device=device)
    tensors = _tensors(batch, device)
    stream = torch.cuda.current_stream(device)
    ev = time_decode(tensors, steps, warmup, stream)
    run_decode_loop(tensors, ev, stream)
    torch.cuda.synchronize()
    step_ms = ev[0][0].elapsed_time(ev[-1][2]) / steps
    kern_ms = statistics.mean(e1.elapsed_time(e2) for _, e1, e2 in ev)
    nbytes = decode_bytes(batch.context_lens, w.num_q_heads, w.num_kv_heads, w.head_dim)
    res = {"gbps": round(nbytes / (step_ms * 1e-3) / 1e9, 1),
           "steps_per_s": round(1e3 / step_ms, 1), "ms_per_step": round(step_ms, 4),
           "attention_kernel_gbps": round(nbytes / (kern_ms * 1e-3) / 1e9, 1)}
    del batch, tensors
    torch.cuda.empty_cache()
    return res


def _tensors(batch, device):
    w = batch.workload
    q = batch.q.to(device)
    k = batch.k_pages.to(device)
    v = batch.v_pages.to(device)
    bt = torch.from_numpy(batch.block_table).to(device)
    cl = torch.from_numpy(batch.context_lens).to(device)
    out = torch.empty_like(q)
    lse = torch.empty((len(batch.context_lens), w.num_q_heads), dtype=torch.float32,
                      device=device)
    ws = torch.empty(cadkv.decode_attention_workspace_size(len(batch.context_lens), w.num_q_heads,
                                                           w.num_kv_heads, w.head_dim,
                                                           bt.shape[1]),
                     dtype=torch.uint8, device=device)
    return q, k, v, bt, cl, out, lse, ws


# ------------------------------------------------------------------ main

def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=400)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload",
                    choices=sorted(DECODE_WORKLOADS) + ["staging", "landscape", "prefill"],
                    default="mixed",
                    help="decode workload of the headline line, or 'staging' to time "
                         "only prefix staging")
    ap.add_argument("--staging-layers", type=int, default=None,
                    help="layers per chunk of the 48-layer staging job (default: the "
                         "largest that fits in device memory)")
    ap.add_argument("--staging-batch", type=int, default=None)
    ap.add_argument("--landscape-batches", type=str, default=None,
                    help="landscape: comma-separated batch sizes (default: the whole grid, "
                         "with the composition cells)")
    ap.add_argument("--landscape-means", type=str, default=None,
                    help="landscape: comma-separated mean context lengths")
    ap.add_argument("--cpu-seconds", type=float, default=12.0,
                    help="target oracle time of the cpu_baseline sample")
    ap.add_argument("--reference-seconds", type=float, default=90.0,
                    help="target total oracle time of the --impl reference run")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extras", action="store_true",
                    help="skip the staging and other-workload secondary measurements")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")

    world, rank, local = dist_setup(args)
    if args.impl == "reference":
        return reference_arm(args, world, rank)

    pkg_build.build()
    device = torch.device("cuda", torch.cuda.current_device())
    if args.workload == "staging":
        host = bench_host_staging(device, reps=args.steps)
        res = bench_staging(device, chunk_layers=args.staging_layers,
                            batch=args.staging_batch, cpu_baseline=not args.no_cpu_baseline)
        res["host"] = host
        if rank == 0:
            print(json.dumps(res), flush=True)
        return
    if args.workload == "prefill":
        res = bench_prefill(device, args.steps, args.warmup, cpu_baseline=not args.no_cpu_baseline)
        if rank == 0:
            print(json.dumps(res), flush=True)
        return
    if args.workload == "landscape":
        # Composition cells (0.5-2 GB each) first, then the grid, whose cells grow
        # in size: no cell is allocated right after a much larger one was freed,
        # which left the next allocation's reads up to 30 % slower on this GPU.
        grid = {}
        if args.landscape_batches:
            grid["batches"] = tuple(int(x) for x in args.landscape_batches.split(","))
        if args.landscape_means:
            grid["means"] = tuple(int(x) for x in args.landscape_means.split(","))
        comp = [] if grid else bench_composition(device, args.steps, args.warmup)
        cells = bench_landscape(device, args.steps, args.warmup, **grid)
        if rank == 0:
            print(json.dumps({"workload": "decode-throughput landscape over (B, mean context), "
                                          "32/8 heads, D=128, lengths U[C/2, 3C/2]; and over the "
                                          "within-batch length composition at fixed (B, mean context)",
                              "unit": "GB/s", "cells": cells, "composition_cells": comp}), flush=True)
        return
    w = DECODE_WORKLOADS[args.workload]
    batch = make_decode_batch(w, device=device, seed=w.seed + rank)
    tensors = _tensors(batch, device)
    stream = torch.cuda.current_stream(device)
    nbytes = decode_bytes(batch.context_lens, w.num_q_heads, w.num_kv_heads, w.head_dim)

    ev = time_decode(tensors, args.steps, args.warmup, stream)
    sampler = ClockSampler(device)
    barrier(world)
    torch.cuda.synchronize()
    sampler.start()
    run_decode_loop(tensors, ev, stream)
    torch.cuda.synchronize()
    barrier(world)
    clocks = sampler.stop()
    status = cadkv.decode_attention_status(tensors[7])

    total_ms = ev[0][0].elapsed_time(ev[-1][2])
    kern_ms = statistics.mean(e1.elapsed_time(e2) for _, e1, e2 in ev)
    plan_ms = statistics.mean(e0.elapsed_time(e1) for e0, e1, _ in ev)
    total_ms = max_over_ranks(total_ms, world)
    step_ms = total_ms / args.steps
    all_bytes = sum_over_ranks(float(nbytes), world)
    value = all_bytes * args.steps / (total_ms * 1e-3) / 1e9

    append = time_append_step(batch, tensors, max(args.steps // 4, 20), 3, stream)
    e2e_s, h2d, d2h = e2e_loop(batch, tensors, max(args.steps // 4, 20), 3, stream)
    e2e_s = max_over_ranks(e2e_s, world)
    e2e_value = all_bytes / e2e_s / 1e9

    peak, kind = hbm_peak()
    achieved = nbytes / (kern_ms * 1e-3) / 1e9
    read_gbps = read_probe(batch.k_pages)
    line = {
        "metric": METRIC,
        "value": round(value, 1),
        "unit": "GB/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(step_ms, 4),
        "steps_per_s": round(1e3 / step_ms, 2),
        "pct_of_8tbps": round(100 * value / world / NOMINAL_HBM_GBS, 2),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic",
        "config": {"workload": w.name, "batch": len(batch.context_lens),
                   "context_lens": "lognormal median 4096 sigma 1.0 clipped [512, 131072]"
                   if args.workload == "mixed" else str(w.length_args),
                   "total_context_tokens": int(batch.context_lens.sum()),
                   "num_q_heads": w.num_q_heads, "num_kv_heads": w.num_kv_heads,
                   "head_dim": w.head_dim, "page_size": 16,
                   "kv_pool_gb": round(2 * batch.k_pages.numel() * 2 / 1e9, 2),
                   "bytes_per_step": nbytes, "layers_per_step": 1,
                   "l2": "inputs larger than L2 (no flush)",
                   "parallelism": f"replicas x{world}" if world > 1 else "single GPU"},
        "e2e": {"value": round(e2e_value, 1), "unit": "GB/s",
                "ms_per_step": round(e2e_s * 1e3, 4),
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
        "gpu_launches": 2 * args.steps,  # plan + attention per timed step
        "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak,
                     "unit": "GB/s", "frac": round(achieved / peak, 4),
                     "peak_kind": kind, "kernel": "decode_attention_kernel<128>",
                     "kernel_ms": round(kern_ms, 4), "planner_ms": round(plan_ms, 4),
                     "read_probe_gbps": round(read_gbps, 1),
                     "frac_of_read_probe": round(achieved / read_gbps, 4),
                     "traffic": profiled_traffic(PROFILE_SUMMARY, KERNEL_SOURCE)},
        "decode_step_with_append": append,
        "clocks": clocks,
        "device_status": status,
    }
    if rank == 0 and not args.no_extras:
        extras = {}
        for other in ("paced", "long_tail"):
            if other != args.workload:
                extras[other] = bench_config(other, device, max(args.steps // 4, 50), 5)
        line["other_workloads"] = extras
    if rank == 0 and not args.no_cpu_baseline:
        sample = OracleSample(batch, args.cpu_seconds)
        secs = sample.run()
        line["cpu_baseline"] = {"value": round(sample.nbytes / secs / 1e9, 4), "unit": "GB/s",
                                "cores": sample.threads, "kind": "oracle",
                                "sample": sample.desc, "seconds": round(secs, 2)}
    del batch, tensors
    torch.cuda.empty_cache()
    if rank == 0 and not args.no_extras:
        # The 48-layer staging job frees ~230 GB at its end; an allocation made right
        # after a much larger free runs slower on this GPU, so it comes last.
        line["prefill"] = bench_prefill(device, 10, 3, cpu_baseline=not args.no_cpu_baseline)
        host = bench_host_staging(device, reps=5)
        line["staging"] = bench_staging(device, chunk_layers=args.staging_layers,
                                        cpu_baseline=not args.no_cpu_baseline)
        line["staging"]["host"] = host
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def reference_arm(args, world, rank):
    """The oracle, as it stands, on the host cores: same metric and workload,
    each step one oracle evaluation of a bounded sample of the same batch,
    sized so that warm-up plus timed steps take about --reference-seconds."""
    if rank != 0:
        return
    w = DECODE_WORKLOADS[args.workload]
    device = torch.device("cuda", 0) if torch.cuda.is_available() else torch.device("cpu")
    batch = make_decode_batch(w, device=device)
    per_step = min(max(args.reference_seconds / (args.steps + args.warmup), 0.02), 10.0)
    sample = OracleSample(batch, per_step)
    for _ in range(args.warmup):
        sample.run()
    secs = sum(sample.run() for _ in range(args.steps))
    value = sample.nbytes * args.steps / secs / 1e9
    line = {"metric": METRIC, "value": round(value, 4), "unit": "GB/s", "impl": "reference",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(1e3 * secs / args.steps, 2),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic",
            "config": {"workload": w.name, "batch": len(batch.context_lens),
                       "num_q_heads": w.num_q_heads, "num_kv_heads": w.num_kv_heads,
                       "head_dim": w.head_dim, "page_size": 16},
            "cpu_baseline": {"value": round(value, 4), "unit": "GB/s", "cores": sample.threads,
                             "kind": "oracle", "sample": "per step: " + sample.desc},
            "e2e": {"value": round(value, 4), "unit": "GB/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
