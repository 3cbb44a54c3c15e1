#!/usr/bin/env python
"""Benchmark of the paged-attention hot path on one GB300 (or N replicas).

One step = one pass of the whole path over one synthetic batch: KV append of
every query token's new K/V, then paged attention (device planner, cascade
pass over shared GRPO prompts, split-KV decode, causal append-chunk kernel,
log-sum-exp merge) -- for every layer of the workload.

Default workload: the mixed multi-turn batch (256 trajectories with prior
context uniform in [4096, 32768]; 224 decode one token, 32 append a tool
observation of log-uniform length in [64, 2048]; 64 q / 8 kv heads, head dim
64, page 16, bf16). Inputs are resident in HBM when timing starts and are far
larger than L2 (the KV pool alone is ~10 GB), so no L2 flush is needed.

Metric: KV-read GB/s = algorithmic KV bytes per step / step time, where the
algorithmic KV bytes count every (row, key position) that some query of the
row may see once (shared prompt pages once per group): 2 * H_kv * D * 2 bytes
per token. Attended tokens/s (sum over queries of visible keys) is reported
beside it.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                  [--workload mixed|decode|long|rollout|tiny|mixed_small|rollout_small|churn]
                  [--kv bf16|fp8] [--launch graph|eager]

Prints one JSON line (rank 0). Under torchrun each rank runs an independent
replica on its own GPU (the path has no exchange step); value is the total
over ranks divided by the slowest rank's time.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import threading
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import workloads as W  # noqa: E402

KV_TOKEN_BYTES = lambda b: 2 * b.num_kv_heads * b.head_dim * 2  # noqa: E731
WORKLOAD_DESC = {
    "tiny": "tiny decode: 4 rows, S={17,64,129,300}, 8q/2kv heads, D=64, page 16, bf16",
    "decode": "decode batch: 64 rows, S~U[2048,16384], 64q/8kv, D=64, page 16, bf16",
    "mixed": "mixed multi-turn batch: 256 rows, prior~U[4096,32768], 224 decode + 32 append rows "
             "(chunk logU[64,2048]), 64q/8kv, D=64, page 16, bf16",
    "mixed_small": "mixed batch at 64 rows (8 append), same distributions; profiling case",
    "long": "long-horizon decode: 512 rows, S lognormal(median 12288, sigma 1) in [512,65536], "
            "1/3 in [49152,65536], 64q/8kv, D=64, page 16, bf16",
    "rollout": "rollout step: 24 layers alternating SWA-128/full, 48 GRPO groups x 8 rows sharing prompt "
               "pages (prompt U[1024,8192], continuation U[0,24576]), 15% append rows (logU[64,1024]), "
               "64q/8kv, D=64, page 16, bf16",
    "rollout_small": "rollout step at 8 GRPO groups x 8 rows and 4 layers (SWA-128/full alternating), same "
                     "distributions; profiling case",
}


def recorded_traffic(kernel_md: str, key: str, sources):
    """DRAM bytes per launch recorded in a profiles/ summary, or None when the
    kernel's sources changed since the capture (sha256 mismatch)."""
    import hashlib
    import re

    path = os.path.join(ROOT, "profiles", kernel_md)
    try:
        text = open(path).read()
        h = hashlib.sha256()
        for f in sources:
            h.update(open(os.path.join(ROOT, f), "rb").read())
        sha = re.search(r"source_sha256: ([0-9a-f]{64})", text).group(1)
        val = re.search(key + r": (\d+)", text).group(1)
        return int(val) if sha == h.hexdigest() else None
    except Exception:
        return None


APPEND_TC_SOURCES = [
    "paper_2608_22167_gb300/csrc/append_tc.cu",
    "paper_2608_22167_gb300/csrc/tcgen05.cuh",
    "paper_2608_22167_gb300/csrc/common.cuh",
    "paper_2608_22167_gb300/csrc/plan.cu",  # item order and split lengths shape the traffic
]
DECODE_SOURCES = [
    "paper_2608_22167_gb300/csrc/decode.cu",
    "paper_2608_22167_gb300/csrc/common.cuh",
    "paper_2608_22167_gb300/csrc/plan.cu",
]
FP8_SOURCES = [
    "paper_2608_22167_gb300/csrc/fp8.cu",
    "paper_2608_22167_gb300/csrc/common.cuh",
    "paper_2608_22167_gb300/csrc/plan.cu",
]
FP8_WORKLOADS = ("tiny", "decode", "long")
NOMINAL_HBM_GBS = 8000.0  # the nominal HBM3e figure the targets are also quoted against


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        sustained = float(d.get("bf16_tflops_sustained", d["bf16_tflops"]))
        return float(d["hbm_gbs"]), float(d["bf16_tflops"]), sustained, "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


# ------------------------------------------------------------------ ranks


def max_over_ranks(values, device, world: int):
    """Element-wise maximum of per-rank timings over all ranks (the slowest
    rank decides); unchanged when running alone."""
    if world <= 1:
        return [float(v) for v in values]
    t = torch.tensor([float(v) for v in values], device=device, dtype=torch.float64)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return [float(x) for x in t.tolist()]


def whole_job_gbs(bytes_per_rank: int, world: int, ms: float) -> float:
    """Throughput of all replicas together: every rank processed its own
    bytes_per_rank in at most `ms`."""
    return bytes_per_rank * world / (ms * 1e-3) / 1e9


# --------------------------------------------------------------- accounting


def kv_token_bytes(batch: W.Batch, kv: str = "bf16") -> int:
    """KV bytes one token occupies over all kv heads: bf16 K and V rows, or
    e4m3 codes plus one float scale per row."""
    if kv == "fp8":
        return 2 * batch.num_kv_heads * (batch.head_dim + 4)
    return KV_TOKEN_BYTES(batch)


def layer_stats(batch: W.Batch, layer: int, kv: str = "bf16"):
    """Algorithmic work of one layer: KV bytes (distinct visible tokens, shared
    prompt pages once per group), attended (query, key) pairs, split by
    decode / append rows."""
    lay = batch.layers[layer]
    Wn = lay.sliding_window
    S = batch.seq_lens.astype(np.int64)
    L = batch.q_lens.astype(np.int64)
    first = np.where(Wn > 0, np.maximum(0, S - L - Wn + 1), 0) if Wn > 0 else np.zeros_like(S)
    distinct = np.where(L > 0, S - first, 0)
    # attended pairs per row: sum_i min(p_i + 1, W)
    pairs = np.zeros_like(S)
    for r in range(len(S)):
        if L[r] == 0:
            continue
        p = np.arange(S[r] - L[r], S[r])
        vis = p + 1 if Wn <= 0 else np.minimum(p + 1, Wn)
        pairs[r] = int(vis.sum())
    shared_tokens = 0
    if Wn <= 0 and batch.group_of_row is not None:
        bt = batch.pools[lay.pool].block_table
        for g in np.unique(batch.group_of_row):
            rows = np.nonzero(batch.group_of_row == g)[0]
            rows = rows[L[rows] > 0]
            if len(rows) < 2:
                continue
            n = 0
            ref = bt[rows[0]]
            lim = int(min(S[rows]) // batch.page_size)
            while n < lim and all(bt[r, n] == ref[n] for r in rows):
                n += 1
            shared_tokens += (len(rows) - 1) * n * batch.page_size
    tb = kv_token_bytes(batch, kv)
    dec = L == 1
    app = L > 1
    return dict(
        kv_bytes=int((distinct.sum() - shared_tokens) * tb),
        kv_bytes_decode=int(distinct[dec].sum() * tb),
        kv_bytes_append=int(distinct[app].sum() * tb),
        shared_tokens_saved=int(shared_tokens),
        pairs=int(pairs.sum()),
        pairs_decode=int(pairs[dec].sum()),
        pairs_append=int(pairs[app].sum()),
        flops_append=int(pairs[app].sum()) * 4 * batch.head_dim * batch.num_q_heads,
        flops=int(pairs.sum()) * 4 * batch.head_dim * batch.num_q_heads,
    )


# ------------------------------------------------------------------- clocks


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 100 ms in the background."""

    FIELDS = ("index,uuid,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid: str | None):
        self.uuid = uuid
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader",
                                          "-lms", "100"], stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        rows = []
        with open(self.path) as f:
            for line in f:
                c = [x.strip() for x in line.split(",")]
                if len(c) < 10:
                    continue
                if self.uuid and self.uuid not in c[1]:
                    continue
                rows.append(c)
        os.unlink(self.path)
        if not rows:
            return None

        def mhz(x):
            try:
                return float(x.split()[0])
            except Exception:
                return float("nan")

        sm = [mhz(r[2]) for r in rows]
        reasons = set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            for n, v in zip(names, r[6:10]):
                if v.strip().lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mhz(r[3]) for r in rows),
                "reasons": sorted(reasons), "samples": len(rows)}


# ------------------------------------------------------------------ our arm


class Stepper:
    """Device-resident inputs of every layer and one call sequence per step."""

    def __init__(self, batch: W.Batch, dev):
        from paper_2608_22167_gb300 import mcpu

        self.mcpu = mcpu
        self.batch = batch
        self.dev = dev
        self.sl = torch.from_numpy(batch.seq_lens).to(dev)
        self.qsl = torch.from_numpy(batch.query_start_loc).to(dev)
        self.bts = {k: torch.from_numpy(p.block_table).to(dev) for k, p in batch.pools.items()}
        self.layers = batch.layers
        lay0 = batch.layers[0]
        p0 = batch.pools[lay0.pool]
        self.dims = mcpu.dims(lay0.q, p0.k_cache, self.bts[lay0.pool], self.sl)
        self.ws = mcpu.new_workspace(self.dims, dev)
        self.out = torch.empty_like(lay0.q)
        self.lse = torch.empty(lay0.q.shape[:2], dtype=torch.float32, device=dev)
        self.launches_per_layer = {}
        for i, lay in enumerate(batch.layers):
            cascade = 1 if lay.sliding_window <= 0 else 0
            # KV append, [prefix scan], plan, decode, [cascade], append chunks, merge
            self.launches_per_layer[i] = 5 + 2 * cascade

    def layer_call(self, i, q=None, k_new=None, v_new=None, out=None, lse=None, events=None):
        m = self.mcpu
        lay = self.layers[i]
        pool = self.batch.pools[lay.pool]
        bt = self.bts[lay.pool]
        m.mcpu_kv_append(lay.k_new if k_new is None else k_new, lay.v_new if v_new is None else v_new,
                         pool.k_cache, pool.v_cache, bt, self.sl, self.qsl, m.status_word(self.ws))
        m.mcpu_paged_attention_forward(lay.q if q is None else q, pool.k_cache, pool.v_cache, bt, self.sl, self.qsl,
                                       lay.sliding_window, self.batch.softmax_scale,
                                       self.out if out is None else out, self.lse if lse is None else lse,
                                       self.ws, phase_events=events)

    def step(self, events=None):
        for i in range(len(self.layers)):
            self.layer_call(i, events=None if events is None else events[i])

    @property
    def launches_per_step(self):
        return sum(self.launches_per_layer.values())


def quantize_pools_fp8(batch: W.Batch, dev):
    """An fp8 pool (uint8 [P, Hkv, 2176]) for every bf16 pool, written by
    mcpu_kv_append_fp8 with every page appended as one 16-token row (input
    preparation, untimed)."""
    from paper_2608_22167_gb300 import mcpu

    status = torch.zeros(1, dtype=torch.int32, device=dev)
    pools = {}
    for key, pool in batch.pools.items():
        P, H, page, D = pool.k_cache.shape
        kv8 = mcpu.new_fp8_pool(P, H, dev)
        chunk = 2048  # rows per call (the planner's row limit)
        for p0 in range(0, P, chunk):
            n = min(chunk, P - p0)
            kn = pool.k_cache[p0:p0 + n].permute(0, 2, 1, 3).reshape(n * page, H, D).contiguous()
            vn = pool.v_cache[p0:p0 + n].permute(0, 2, 1, 3).reshape(n * page, H, D).contiguous()
            bt = torch.arange(p0, p0 + n, dtype=torch.int32, device=dev).view(n, 1)
            sl = torch.full((n,), page, dtype=torch.int32, device=dev)
            qsl = torch.arange(0, (n + 1) * page, page, dtype=torch.int32, device=dev)
            mcpu.mcpu_kv_append_fp8(kn, vn, kv8, bt, sl, qsl, status)
        pools[key] = kv8
    torch.cuda.synchronize()
    if int(status.item()) != 0:
        raise RuntimeError(f"fp8 pool quantization: device status {int(status.item())}")
    return pools


class Fp8Stepper(Stepper):
    """The same step over fp8 KV pages: quantizing KV append, then the fp8
    forward (decode rows only)."""

    def __init__(self, batch: W.Batch, dev):
        super().__init__(batch, dev)
        self.pools8 = quantize_pools_fp8(batch, dev)
        for i, lay in enumerate(batch.layers):
            # KV append, [prefix scan], plan, decode, [cascade], merge
            self.launches_per_layer[i] = 4 + 2 * (1 if lay.sliding_window <= 0 else 0)

    def layer_call(self, i, q=None, k_new=None, v_new=None, out=None, lse=None, events=None):
        m = self.mcpu
        lay = self.layers[i]
        kv8 = self.pools8[lay.pool]
        bt = self.bts[lay.pool]
        m.mcpu_kv_append_fp8(lay.k_new if k_new is None else k_new, lay.v_new if v_new is None else v_new,
                             kv8, bt, self.sl, self.qsl, m.status_word(self.ws))
        m.mcpu_paged_attention_forward_fp8(lay.q if q is None else q, kv8, bt, self.sl, self.qsl, lay.sliding_window,
                                           self.batch.softmax_scale, self.out if out is None else out,
                                           self.lse if lse is None else lse, self.ws, phase_events=events)


def make_batch(name, dev, rank):
    fn = W.CONFIGS[name]
    seed = {"tiny": 1001, "decode": 1002, "mixed": 1003, "mixed_small": 1013, "long": 1004,
            "rollout": 1005, "rollout_small": 1015}[name] + 7 * rank
    return fn(seed=seed, device=dev)


def oracle_fp8_pools(k_bits, v_bits):
    """A (compact, host) bf16 pool quantized by the oracle, every page
    appended as one 16-token row: (k8, v8, k_scale, v_scale), V row-major."""
    import oracle

    P, H, page, D = k_bits.shape
    tok = lambda x: np.ascontiguousarray(x.transpose(0, 2, 1, 3).reshape(P * page, H, D))  # noqa: E731
    z8 = np.zeros((P, H, page, D), np.uint8)
    zs = np.zeros((P, H, page), np.float32)
    return oracle.kv_append_fp8(tok(k_bits), tok(v_bits), z8, z8, zs, zs, np.arange(P, dtype=np.int32)[:, None],
                                np.full(P, page, np.int32), np.arange(P + 1, dtype=np.int32) * page)


def cpu_model() -> str:
    """The host CPU's name (x86 'model name', else the Arm implementer/part)."""
    try:
        info = open("/proc/cpuinfo").read()
    except OSError:
        return "unknown"
    for line in info.splitlines():
        if line.lower().startswith("model name"):
            return line.split(":", 1)[1].strip()
    parts = {"0x41": "Arm", "0x4e": "NVIDIA"}
    impl = part = None
    for line in info.splitlines():
        if line.startswith("CPU implementer") and impl is None:
            impl = line.split(":", 1)[1].strip()
        if line.startswith("CPU part") and part is None:
            part = line.split(":", 1)[1].strip()
    names = {"0xd4f": "Neoverse-V2"}
    return f"{parts.get(impl, impl)} {names.get(part, part)}" if impl else "unknown"


def cpu_baseline_sample(batch: W.Batch, stats_total, seconds: float, seed: int, kv: str = "bf16"):
    """Time the oracle on a bounded sample of the workload and scale its
    throughput to the whole step by attended (query, key) pairs."""
    import oracle

    rng = np.random.default_rng(seed)
    L = batch.q_lens
    dec = np.nonzero(L == 1)[0]
    app = np.nonzero(L > 1)[0]
    t_spent = 0.0
    pairs_done = 0
    n_tok = 0
    rounds = 0
    Wn = batch.layers[0].sliding_window
    while t_spent < seconds and rounds < 50:
        rounds += 1
        rows = list(rng.choice(dec, size=min(6, len(dec)), replace=False)) if len(dec) else []
        if len(app):
            rows += list(rng.choice(app, size=min(2, len(app)), replace=False))
        h = W.host_rows(batch, rows, 0)
        if kv == "fp8":
            pools8 = oracle.kv_append_fp8(h["k_new"], h["v_new"], *oracle_fp8_pools(h["k_cache"], h["v_cache"]),
                                          h["block_table"], h["seq_lens"], h["query_start_loc"])
        else:
            kc, vc = oracle.kv_append(h["k_new"], h["v_new"], h["k_cache"], h["v_cache"], h["block_table"],
                                      h["seq_lens"], h["query_start_loc"])
        qsl = h["query_start_loc"]
        toks = []
        for i in range(len(h["rows"])):
            t0, t1 = int(qsl[i]), int(qsl[i + 1])
            sel = np.arange(t0, t1)
            if len(sel) > 24:
                sel = rng.choice(sel, size=24, replace=False)
            toks += list(sel)
        toks = np.asarray(toks, np.int64)
        tk = np.repeat(toks, batch.num_q_heads)
        hd = np.tile(np.arange(batch.num_q_heads, dtype=np.int32), len(toks))
        # attended pairs of the sampled queries
        row_of = np.searchsorted(qsl, toks, side="right") - 1
        S = h["seq_lens"][row_of].astype(np.int64)
        Lr = (qsl[row_of + 1] - qsl[row_of]).astype(np.int64)
        p = S - Lr + (toks - qsl[row_of])
        vis = p + 1 if Wn <= 0 else np.minimum(p + 1, Wn)
        t = time.perf_counter()
        if kv == "fp8":
            oracle.paged_attention_sampled_fp8(h["q"], *pools8, h["block_table"], h["seq_lens"], qsl, Wn,
                                               batch.softmax_scale, tk, hd)
        else:
            oracle.paged_attention_sampled(h["q"], kc, vc, h["block_table"], h["seq_lens"], qsl, Wn,
                                           batch.softmax_scale, tk, hd)
        t_spent += time.perf_counter() - t
        pairs_done += int(vis.sum()) * batch.num_q_heads
        n_tok += len(toks)
    pairs_total = stats_total["pairs"] * batch.num_q_heads
    est_step_s = t_spent * pairs_total / max(pairs_done, 1)
    return dict(
        value=stats_total["kv_bytes"] / est_step_s / 1e9,
        unit="GB/s",
        cores=int(oracle.max_threads()),
        cpu_model=cpu_model(),
        kind="oracle",
        sample=f"{'fp8 pages, ' if kv == 'fp8' else ''}"
               f"{n_tok} query tokens x {batch.num_q_heads} heads from {rounds} draws of 6 decode + 2 append "
               f"rows (layer 0), {t_spent:.1f} s of oracle time; step time scaled by attended (query, key) pairs "
               f"({pairs_done:.3g} of {pairs_total:.3g})",
        est_step_ms=est_step_s * 1e3,
        attended_tokens_per_s=stats_total["pairs"] / est_step_s,
    )


def run_ours(args, rank, world, dev):
    from paper_2608_22167_gb300 import mcpu

    hbm, tc_burst, tc_sust, peak_src = peaks()
    fp8 = args.kv == "fp8"
    if fp8 and args.workload not in FP8_WORKLOADS:
        raise SystemExit(f"--kv fp8 runs decode-only workloads: {', '.join(FP8_WORKLOADS)}")
    batch = make_batch(args.workload, dev, rank)
    st = Fp8Stepper(batch, dev) if fp8 else Stepper(batch, dev)
    per_layer = [layer_stats(batch, i, args.kv) for i in range(len(batch.layers))]
    kv_bytes = sum(s["kv_bytes"] for s in per_layer)
    pairs = sum(s["pairs"] for s in per_layer)

    # warm-up (also the first call performs the per-device setup)
    for _ in range(args.warmup):
        st.step()
    torch.cuda.synchronize()
    code, bits = mcpu.mcpu_read_device_status(st.ws)
    if code != 0:
        raise RuntimeError(f"device status {bits} after warm-up")

    nl = len(batch.layers)
    stream = torch.cuda.current_stream()
    # The timed steps record nothing but the start and end events (event
    # records captured in a graph cost device time at every replay). The
    # per-kernel spans come from separate, untimed steps that record the
    # phase events: one set per step (eager) or per captured graph (each
    # graph records its own set at every replay).
    n_sets = min(args.steps, 16)
    phase = [[[torch.cuda.Event(enable_timing=True) for _ in range(mcpu.NUM_PHASE_EVENTS)] for _ in range(nl)]
             for _ in range(n_sets)]
    for s in phase:  # create the events (torch creates them lazily)
        for lay in s:
            for e in lay:
                e.record(stream)
    graphs = []
    g_timed = None
    if args.launch == "graph":
        # the whole step (every layer's KV append and forward) as CUDA graphs;
        # the planner runs inside the graph, so nothing is precomputed
        g_timed = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g_timed):
            st.step()
        for j in range(n_sets):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                st.step(events=phase[j])
            graphs.append(g)
        g_timed.replay()  # upload, untimed
        for g in graphs:
            g.replay()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    uuid = None
    try:
        uuid = str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:
        pass
    sampler = ClockSampler(uuid)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    sampler.start()
    time.sleep(0.3)  # let the sampler start before the timed region
    wall0 = time.perf_counter()
    t_start.record(stream)
    for k in range(args.steps):
        if g_timed is not None:
            g_timed.replay()
        else:
            st.step()
    t_end.record(stream)
    torch.cuda.synchronize()
    wall = time.perf_counter() - wall0
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    clocks = sampler.stop()
    total_ms = float(t_start.elapsed_time(t_end))
    code, bits = mcpu.mcpu_read_device_status(st.ws)
    if code != 0:
        raise RuntimeError(f"device status {bits} in the timed region")

    # the instrumented steps behind the per-kernel spans (untimed)
    for k in range(n_sets):
        if graphs:
            graphs[k].replay()
        else:
            st.step(events=phase[k])
    torch.cuda.synchronize()

    # the other launch mode, same steps, for comparison (untimed for `value`)
    other_ms = None
    if args.compare_launch:
        torch.cuda.synchronize()
        o0 = torch.cuda.Event(enable_timing=True)
        o1 = torch.cuda.Event(enable_timing=True)
        n_other = min(args.steps, 50)
        if graphs:
            o0.record(stream)
            for k in range(n_other):
                st.step()
            o1.record(stream)
        else:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                st.step()
            g.replay()
            o0.record(stream)
            for k in range(n_other):
                g.replay()
            o1.record(stream)
        torch.cuda.synchronize()
        other_ms = o0.elapsed_time(o1) / n_other

    # per-kernel times, ms per step. Decode, cascade and merge run in that
    # order on the library's side stream concurrently with the append
    # kernel: events [1]->[2] decode, [2]->[3] cascade (side stream), [1]->[4]
    # append, [5] after the join; "merge" is the time from the later of [3]
    # and [4] to [5], what the merge (and the join) add past both.
    ktime = {n: 0.0 for n in ("plan", "decode", "cascade", "append_chunk", "merge")}
    layer_ms = [0.0] * nl  # each layer's forward span (planner to merge)
    layer_k = [[0.0] * 5 for _ in range(nl)]  # plan, decode+cascade, append, merge (past both), total
    for k in range(n_sets):
        for i in range(nl):
            ev = phase[k][i]
            t = [0.0] + [ev[0].elapsed_time(ev[j]) for j in range(1, len(ev))]
            layer_ms[i] += t[5] / n_sets
            for j, v in enumerate((t[1], t[3] - t[1], t[4] - t[1], t[5] - max(t[3], t[4]), t[5])):
                layer_k[i][j] += v / n_sets
            ktime["plan"] += t[1]
            ktime["decode"] += t[2] - t[1]
            ktime["cascade"] += t[3] - t[2]
            if fp8:  # one stream, no append kernel: [3] and [4] coincide
                ktime["merge"] += t[5] - t[4]
            else:
                ktime["append_chunk"] += t[4] - t[1]
                ktime["merge"] += t[5] - max(t[3], t[4])
    ktime = {n: v / n_sets for n, v in ktime.items()}
    dec_bytes = sum(s["kv_bytes"] - s["kv_bytes_append"] for s in per_layer)
    app_flops = sum(s["flops_append"] for s in per_layer)
    dec_ms = ktime["cascade"] + ktime["decode"]
    app_ms = ktime["append_chunk"]
    roof_dec = None
    if dec_ms > 0 and dec_bytes > 0:
        ach = dec_bytes / (dec_ms * 1e-3) / 1e9
        traffic = None
        if args.workload in ("decode", "long"):
            if fp8:
                traffic = recorded_traffic("decode_fp8_kernel_decode_long.md",
                                           f"traffic_bytes_per_launch_{args.workload}", FP8_SOURCES)
            else:
                traffic = recorded_traffic("decode_kernel_decode_long.md",
                                           f"traffic_bytes_per_launch_{args.workload}", DECODE_SOURCES)
        roof_dec = {"bound": "hbm", "achieved": round(ach, 1), "peak": hbm, "unit": "GB/s",
                    "frac": round(ach / hbm, 4), "traffic": traffic,
                    "kernel": ("decode_fp8_kernel" if fp8 else "decode_kernel") + " (+cascade pass)",
                    "peak_source": f"{peak_src} hbm_gbs", "ms_per_step": round(dec_ms, 4)}
    roof_app = None
    if app_ms > 0 and app_flops > 0:
        ach = app_flops / (app_ms * 1e-3) / 1e12
        traffic = None
        if args.workload == "mixed":
            traffic = recorded_traffic("append_tc_kernel_mixed.md", "traffic_bytes_per_launch_mixed",
                                       APPEND_TC_SOURCES)
        roof_app = {"bound": "tensor", "achieved": round(ach, 2), "peak": tc_burst, "unit": "TFLOP/s",
                    "frac": round(ach / tc_burst, 4), "traffic": traffic,
                    "algorithmic_bytes": int(sum(s["kv_bytes_append"] for s in per_layer)
                                             + 2 * int(batch.q_lens[batch.q_lens > 1].sum()) * batch.num_q_heads
                                             * batch.head_dim * 2),
                    "kernel": "append_tc_kernel",
                    "peak_source": f"{peak_src} bf16_tflops (burst)", "ms_per_step": round(app_ms, 4)}
    cands = [r for r in (roof_dec, roof_app) if r is not None]
    # the kernel that bounds the step: the tensor-core append kernel when the
    # step's flops take longer at the bf16 peak than its KV bytes at the HBM
    # peak (the decode kernels' spans on the side stream then include time
    # spent waiting for SMs the append kernel holds), else the decode kernel
    step_flops = sum(s["flops"] for s in per_layer)
    tensor_bound = step_flops / (tc_burst * 1e12) > sum(s["kv_bytes"] for s in per_layer) / (hbm * 1e9)
    if tensor_bound and roof_app is not None:
        dominant = roof_app
    elif roof_dec is not None:
        dominant = roof_dec
    else:
        dominant = max(cands, key=lambda r: r["ms_per_step"]) if cands else None

    # ---- end to end: host buffers, copies inside the timed region: every
    # layer through mcpu_paged_attention_host (_fp8 over fp8 pools), which
    # copies q / k_new / v_new in and out / lse back, overlapped with the
    # compute by row slices; the step ends when its last output is in host
    # memory.
    e2e_steps = 0 if getattr(args, "skip_e2e", False) else max(3, min(args.steps, 20))
    h2d = d2h = 0
    e2e_ms = e2e_median_ms = float("nan")
    if e2e_steps:
        lay_host = []
        for lay in batch.layers:
            lay_host.append((lay.q.cpu().pin_memory(), lay.k_new.cpu().pin_memory(), lay.v_new.cpu().pin_memory()))
        meta_host = [torch.from_numpy(batch.seq_lens).to(torch.int32).pin_memory(),
                     torch.from_numpy(batch.query_start_loc).to(torch.int32).pin_memory()]
        bt_host = {k: torch.from_numpy(p.block_table).pin_memory() for k, p in batch.pools.items()}
        # each step's block tables go into one of two device copies on a copy
        # stream of their own, so the copy overlaps the previous step instead
        # of queueing on the compute stream behind it (and behind the stage's
        # input copies on the same engine)
        bt_dev = [{k: v.clone() for k, v in st.bts.items()} for _ in range(2)]
        bt_stream = torch.cuda.Stream()
        bt_ready = [torch.cuda.Event(), torch.cuda.Event()]
        bt_free = [torch.cuda.Event(), torch.cuda.Event()]
        e2e_count = [0]
        q0 = batch.layers[0].q
        out_h = torch.empty(q0.shape, dtype=q0.dtype).pin_memory()
        lse_h = torch.empty(q0.shape[:2], dtype=torch.float32).pin_memory()
        h2d = sum(t.numel() * t.element_size() for tr in lay_host for t in tr)
        h2d += sum(t.numel() * t.element_size() for t in meta_host) + sum(
            t.numel() * t.element_size() for t in bt_host.values())
        d2h = (out_h.numel() * out_h.element_size() + lse_h.numel() * 4) * nl
        host_stage = mcpu.HostStage(q0.shape[0], batch.num_seqs, batch.num_q_heads, batch.num_kv_heads, slots=3)

        def e2e_step():
            j = e2e_count[0] % 2
            e2e_count[0] += 1
            bts = bt_dev[j]
            with torch.cuda.stream(bt_stream):
                bt_stream.wait_event(bt_free[j])  # the step two back is done with this copy
                for key, t in bt_host.items():
                    bts[key].copy_(t, non_blocking=True)
                bt_ready[j].record(bt_stream)
            stream.wait_event(bt_ready[j])
            for i in range(nl):
                lay = batch.layers[i]
                qh, knh, vnh = lay_host[i]
                # the step's last layer writes its outputs straight into the
                # page-locked host buffers (they are read back right after
                # it); earlier layers run as one slice each: their copies back
                # run beside the next layers, so cutting them into row slices
                # would only add each slice's planner and kernel tails
                # (rollout: median step 60.7 -> 59.5 ms with one slice)
                last = i == nl - 1
                fl = mcpu.FLAG_HOST_OUT_DIRECT if last else 0
                nsl = 0 if last else 1
                if fp8:
                    mcpu.mcpu_paged_attention_host_fp8(host_stage, qh, knh, vnh, st.pools8[lay.pool], bts[lay.pool],
                                                       meta_host[0], meta_host[1], lay.sliding_window,
                                                       batch.softmax_scale, out_h, lse_h, st.ws, flags=fl,
                                                       slices=nsl)
                else:
                    pool = batch.pools[lay.pool]
                    mcpu.mcpu_paged_attention_host(host_stage, qh, knh, vnh, pool.k_cache, pool.v_cache,
                                                   bts[lay.pool], meta_host[0], meta_host[1], lay.sliding_window,
                                                   batch.softmax_scale, out_h, lse_h, st.ws, flags=fl,
                                                   slices=nsl)
            mcpu.mcpu_host_stage_wait(host_stage)
            bt_free[j].record(stream)

        for _ in range(2):
            e2e_step()
        torch.cuda.synchronize()
        if world > 1:
            torch.distributed.barrier()
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(e2e_steps + 1)]
        ev[0].record(stream)
        for k in range(e2e_steps):
            e2e_step()
            ev[k + 1].record(stream)
        torch.cuda.synchronize()
        e2e_ms = ev[0].elapsed_time(ev[-1]) / e2e_steps
        # per-step spread: host-to-device copies out of a multi-GB page-locked
        # working set can stall for a pass (plain copies do too); the median
        # shows a typical step, the mean (the reported value) includes stalls
        e2e_median_ms = statistics.median(ev[k].elapsed_time(ev[k + 1]) for k in range(e2e_steps))
        mcpu.mcpu_host_stage_sync(host_stage)
        host_stage.close()

    # ---- max over ranks
    total_ms, e2e_ms = max_over_ranks([total_ms, e2e_ms], dev, world)
    ms_per_step = total_ms / args.steps
    # the step's own bound: max(KV bytes / HBM peak, attention flops / bf16 peak)
    flops = sum(s["flops"] for s in per_layer)
    ideal_ms = max(kv_bytes / (hbm * 1e9), flops / (tc_burst * 1e12)) * 1e3
    combined = {"ideal_ms": round(ideal_ms, 4), "frac": round(ideal_ms / ms_per_step, 4),
                "bound": "hbm" if kv_bytes / (hbm * 1e9) >= flops / (tc_burst * 1e12) else "tensor",
                "flops_per_step": int(flops)}
    value = whole_job_gbs(kv_bytes, world, ms_per_step)
    e2e_value = whole_job_gbs(kv_bytes, world, e2e_ms)

    res = {
        "metric": "KV-read HBM GB/s (% of GB300 peak) and attended tokens/s, paged mixed batch",
        "value": round(value, 2),
        "unit": "GB/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(ms_per_step, 4),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "e4m3 KV pages (f16 MMA, f32 softmax), bf16 q/out" if fp8 else "bf16",
        "data": "synthetic (seeded N(0,1) bf16 Q/K/V; lengths drawn per the workload recipe)"
                + ("; the pools quantized to e4m3 with one scale per (token, kv head) row" if fp8 else ""),
        "config": {
            "workload": ("fp8 KV pages, " if fp8 else "") + WORKLOAD_DESC[args.workload],
            "kv": args.kv,
            "layers": nl,
            "rows": batch.num_seqs,
            "query_tokens": batch.total_q,
            "kv_bytes_per_step": kv_bytes,
            "attended_pairs_per_step": pairs,
            "l2": "inputs larger than L2 (KV pool %.1f GB >> 126 MB L2); no flush" % (
                sum(p.k_cache.numel() * (4 if not fp8 else 2 * (batch.head_dim + 4) / batch.head_dim)
                    for p in batch.pools.values()) / 1e9),
            "parallelism": f"replicas x{world} (no exchange step)",
            "launch": "one CUDA graph per step (KV append + forward of every layer)" if graphs
                      else "eager (C-ABI calls per layer)",
        },
        "frac_of_hbm_peak": round(value / world / hbm, 4),
        "frac_of_nominal_hbm": round(value / world / NOMINAL_HBM_GBS, 4),
        "combined_roofline": combined,
        "attended_tokens_per_s": round(pairs * world / (ms_per_step * 1e-3), 1),
        "kernel_ms_per_step": {k: round(v, 4) for k, v in ktime.items()},
        "layer_ms": [round(v, 4) for v in layer_ms] if nl > 1 else None,
        "layer_kernel_ms": ({"plan, decode+cascade, append, merge, total": [
            [round(v, 4) for v in layer_k[i]] for i in range(min(nl, 2))]} if nl > 1 else None),
        ("eager_ms_per_step" if graphs else "graph_ms_per_step"): (round(other_ms, 4) if other_ms else None),
        "roofline": dominant,
        "roofline_decode": roof_dec,
        "roofline_append": roof_app,
        "gpu_launches": st.launches_per_step * args.steps,
        "e2e": None if not e2e_steps else {"value": round(e2e_value, 2), "unit": "GB/s", "h2d_bytes_per_step": int(h2d),
                "d2h_bytes_per_step": int(d2h), "ms_per_step": round(e2e_ms, 4),
                "median_step_ms": round(e2e_median_ms, 4),
                "call": ("mcpu_paged_attention_host_fp8" if fp8 else "mcpu_paged_attention_host") +
                        " per layer (host q/k_new/v_new/out/lse; inputs copied while the previous call computes;"
                        " outputs copied back beside the next layer, one slice each, the last layer's written"
                        " in place)"},
        "clocks": clocks,
        "wall_s_timed": round(wall, 3),
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        stats0 = per_layer[0]
        cb = cpu_baseline_sample(batch, {"kv_bytes": stats0["kv_bytes"], "pairs": stats0["pairs"]},
                                 args.cpu_seconds, seed=99, kv=args.kv)
        res["cpu_baseline"] = {k: (round(v, 4) if isinstance(v, float) else v) for k, v in cb.items()}
    return res


CHURN_DESC = ("rollout simulator: 48 GRPO groups x 8 live trajectories, prompts U[1024,8192] shared per group, "
              "responses logU[16,256] tokens per turn, tool waits U[2,20] steps, observations logU[64,1024], "
              "2-6 turns, max 32768 tokens; 64q/8kv, D=64, page 16, bf16; the batch changes every step")


def churn_config():
    from paper_2608_22167_gb300.rollout_sim import SimConfig

    return SimConfig(num_pages=1 << 20, max_pages_per_seq=2048, max_live_groups=48, group_size=8,
                     prompt_len=(1024, 8192), response_len=(16, 256), observation_len=(64, 1024),
                     tool_wait_steps=(2, 20), acquire_steps=(0, 4), max_turns=(2, 6), max_len=32768)


def run_churn(args, rank, world, dev):
    """The path fed by the rollout simulator: every step the batch changes
    (trajectories join after acquiring an environment, decode, stop on tool
    calls, append observations, finish). The simulator first runs
    `--churn-settle` host-only steps so the timed steps see a settled mix of
    lengths and states; the KV pool is filled with N(0,1) values once."""
    from paper_2608_22167_gb300 import mcpu
    from paper_2608_22167_gb300.rollout_sim import RolloutSim

    hbm, tc_burst, _, peak_src = peaks()
    cfg = churn_config()
    sim = RolloutSim(cfg, seed=2001 + 7 * rank)
    Hq, Hkv, D = 64, 8, 64
    gen = torch.Generator(device=dev)
    gen.manual_seed(2002 + rank)
    kc = torch.randn((cfg.num_pages, Hkv, 16, D), generator=gen, device=dev, dtype=torch.bfloat16)
    vc = torch.randn((cfg.num_pages, Hkv, 16, D), generator=gen, device=dev, dtype=torch.bfloat16)
    max_t = 1 << 16  # query tokens of one step (a prefill of 8192 plus decodes and observations)
    qbuf = torch.randn((max_t, Hq, D), generator=gen, device=dev, dtype=torch.bfloat16)
    knbuf = torch.randn((max_t, Hkv, D), generator=gen, device=dev, dtype=torch.bfloat16)
    vnbuf = torch.randn((max_t, Hkv, D), generator=gen, device=dev, dtype=torch.bfloat16)
    out = torch.empty_like(qbuf)
    lse = torch.empty((max_t, Hq), dtype=torch.float32, device=dev)
    for _ in range(args.churn_settle):
        sim.step()
    stream = torch.cuda.current_stream()

    def one_step(record):
        b = sim.step()
        if b.num_seqs == 0:
            return None
        T = b.total_q
        if T > max_t:
            raise RuntimeError(f"a step with {T} query tokens exceeds the bench's buffers")
        bt = torch.from_numpy(b.block_table).to(dev)
        sl = torch.from_numpy(b.seq_lens).to(dev)
        qsl = torch.from_numpy(b.query_start_loc).to(dev)
        q, kn, vn = qbuf[:T], knbuf[:T], vnbuf[:T]
        d = mcpu.dims(q, kc, bt, sl)
        ws = mcpu.new_workspace(d, dev)
        e0 = e1 = None
        if record:
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
        mcpu.mcpu_kv_append(kn, vn, kc, vc, bt, sl, qsl, mcpu.status_word(ws))
        mcpu.mcpu_paged_attention_forward(q, kc, vc, bt, sl, qsl, 0, 0.125, out[:T], lse[:T], ws)
        if record:
            e1.record(stream)
        # KV bytes: every visible token once, shared prompt pages once per group
        S = b.seq_lens.astype(np.int64)
        kv_tokens = int(S.sum())
        for g in np.unique(b.groups):
            rows = np.nonzero(b.groups == g)[0]
            if len(rows) < 2:
                continue
            ref = b.block_table[rows[0]]
            lim = int(S[rows].min() // 16)
            n = 0
            while n < lim and np.all(b.block_table[rows, n] == ref[n]):
                n += 1
            kv_tokens -= (len(rows) - 1) * n * 16
        L = b.q_lens.astype(np.int64)
        pairs = int((L * (S - L) + L * (L + 1) // 2).sum())  # query i sees S - L + i + 1 keys
        return dict(ws=ws, ev=(e0, e1), kv_bytes=kv_tokens * 2 * Hkv * D * 2, rows=b.num_seqs, T=T,
                    append_rows=int((L > 1).sum()), pairs=pairs)

    for _ in range(args.warmup):
        one_step(False)
    torch.cuda.synchronize()
    recs = []
    wall0 = time.perf_counter()
    for _ in range(args.steps):
        r = one_step(True)
        if r is not None:
            recs.append(r)
    torch.cuda.synchronize()
    wall = time.perf_counter() - wall0
    for r in recs:
        code, bits = mcpu.mcpu_read_device_status(r["ws"])
        if code != 0:
            raise RuntimeError(f"device status {bits}")
    dev_ms = [r["ev"][0].elapsed_time(r["ev"][1]) for r in recs]
    tot_ms = float(sum(dev_ms))
    kv = sum(r["kv_bytes"] for r in recs)
    tot_ms_all = max_over_ranks([tot_ms], dev, world)[0]
    value = whole_job_gbs(kv // max(world, 1), world, tot_ms_all) if world > 1 else kv / (tot_ms * 1e-3) / 1e9
    return {
        "metric": "KV-read HBM GB/s (% of GB300 peak) and attended tokens/s, paged mixed batch",
        "value": round(value, 2),
        "unit": "GB/s",
        "n_gpus": world,
        "steps": len(recs),
        "warmup": args.warmup,
        "ms_per_step": round(tot_ms_all / max(len(recs), 1), 4),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) bf16 Q/K/V; the batch sequence drawn by the rollout simulator)",
        "config": {"workload": CHURN_DESC, "layers": 1, "settle_steps": args.churn_settle,
                   "mean_rows": round(float(np.mean([r["rows"] for r in recs])), 1),
                   "mean_query_tokens": round(float(np.mean([r["T"] for r in recs])), 1),
                   "mean_append_rows": round(float(np.mean([r["append_rows"] for r in recs])), 2),
                   "l2": "KV pool 34 GB >> 126 MB L2; no flush",
                   "parallelism": f"replicas x{world} (no exchange step)",
                   "launch": "eager; device time per step from CUDA events around the C-ABI calls"},
        "frac_of_hbm_peak": round(value / max(world, 1) / hbm, 4),
        "attended_tokens_per_s": round(sum(r["pairs"] for r in recs) / (tot_ms * 1e-3), 1),
        "generated_tokens_per_s": round(sum(r["T"] for r in recs) / (tot_ms * 1e-3), 1),
        "gpu_launches": 6 * len(recs),
        "wall_s_timed": round(wall, 3),
        "peak_source": peak_src,
    }


# The other four configurations, each timed the same way as the headline (CUDA
# graphs of whole steps, events on the launching stream, clocks sampled) but
# for a fixed, short number of steps, so that one default run measures all
# five: (workload, timed steps). No CPU baseline and no end-to-end leg here.
OTHER_CONFIGS = (("tiny", 200), ("decode", 100), ("long", 20), ("rollout", 8))


def other_configs(args, rank, world, dev):
    out = {}
    for name, steps in OTHER_CONFIGS:
        sub = argparse.Namespace(**vars(args))
        sub.workload, sub.steps, sub.warmup = name, steps, 3
        sub.no_cpu_baseline, sub.compare_launch, sub.skip_e2e = True, False, True
        r = run_ours(sub, rank, world, dev)
        rf = r["roofline"] or {}
        out[name] = {"workload": r["config"]["workload"], "value": r["value"], "unit": r["unit"],
                     "ms_per_step": r["ms_per_step"], "steps": steps,
                     "attended_tokens_per_s": r["attended_tokens_per_s"],
                     "frac_of_hbm_peak": r["frac_of_hbm_peak"], "combined_roofline": r["combined_roofline"],
                     "roofline": {k: rf.get(k) for k in ("bound", "kernel", "achieved", "peak", "unit", "frac",
                                                         "traffic", "ms_per_step")},
                     "kernel_ms_per_step": r["kernel_ms_per_step"], "gpu_launches": r["gpu_launches"],
                     "clocks": r["clocks"]}
        del r
        torch.cuda.empty_cache()
    return out


def run_reference(args, rank, world):
    """The oracle (plain CPU definition) timed on the host cores, rank 0 only."""
    if rank != 0:
        return None
    if args.kv == "fp8" and args.workload not in FP8_WORKLOADS:
        raise SystemExit(f"--kv fp8 runs decode-only workloads: {', '.join(FP8_WORKLOADS)}")
    batch = make_batch(args.workload, "cuda" if torch.cuda.is_available() else "cpu", 0)
    stats0 = layer_stats(batch, 0, args.kv)
    nl = len(batch.layers)
    # each step a bounded oracle sample; the whole run near 150 s of oracle time
    per_step = max(0.5, min(8.0, 150.0 / max(1, args.steps + args.warmup)))
    for w in range(args.warmup):
        cpu_baseline_sample(batch, stats0, per_step / 4, seed=1000 + w, kv=args.kv)
    vals, ms = [], []
    cb = None
    for k in range(args.steps):
        cb = cpu_baseline_sample(batch, stats0, per_step, seed=2000 + k, kv=args.kv)
        vals.append(cb["value"])
        ms.append(cb["est_step_ms"] * nl)
    value = float(statistics.mean(vals))
    return {
        "metric": "KV-read HBM GB/s (% of GB300 peak) and attended tokens/s, paged mixed batch",
        "value": round(value, 4),
        "unit": "GB/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(float(statistics.mean(ms)), 2),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f64",
        "data": "synthetic (seeded N(0,1) bf16 Q/K/V; lengths drawn per the workload recipe)",
        "config": {"workload": ("fp8 KV pages, " if args.kv == "fp8" else "") + WORKLOAD_DESC[args.workload],
                   "kv": args.kv, "layers": nl, "rows": batch.num_seqs},
        "impl": "reference",
        "cpu_baseline": {"value": round(value, 4), "unit": "GB/s", "cores": cb["cores"],
                         "cpu_model": cb["cpu_model"], "kind": "oracle", "sample": cb["sample"]},
        "e2e": {"value": round(value, 4), "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=sorted(W.CONFIGS) + ["churn"], default="mixed")
    ap.add_argument("--churn-settle", type=int, default=400,
                    help="host-only simulator steps before the churn workload's first GPU step")
    ap.add_argument("--kv", choices=["bf16", "fp8"], default="bf16",
                    help="KV page format; fp8 (e4m3 + per-row scales) runs decode-only workloads")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--launch", choices=["graph", "eager"], default="graph",
                    help="time CUDA-graph replays of the whole step (default) or eager C-ABI calls")
    ap.add_argument("--no-compare-launch", dest="compare_launch", action="store_false",
                    help="skip timing the other launch mode")
    ap.add_argument("--no-other-configs", dest="other_configs", action="store_false",
                    help="with the default workload on one GPU: skip the short runs of the other four "
                         "configurations that are added to the line under 'configs'")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        torch.cuda.set_device(local)
        torch.distributed.init_process_group("nccl")
    dev = torch.device("cuda", local)

    if args.impl == "reference":
        res = run_reference(args, rank, world)
    else:
        if not torch.cuda.is_available():
            raise SystemExit("bench.py needs a CUDA GPU for --impl ours")
        torch.cuda.set_device(dev)
        from __graft_entry__ import build

        # one compile at most: rank 0 first, the others find it up to date
        if world > 1 and rank != 0:
            torch.distributed.barrier()
        build()
        if world > 1 and rank == 0:
            torch.distributed.barrier()
        res = run_churn(args, rank, world, dev) if args.workload == "churn" else run_ours(args, rank, world, dev)
        if (world == 1 and args.workload == "mixed" and args.kv == "bf16" and args.other_configs
                and args.launch == "graph"):
            res["configs"] = other_configs(args, rank, world, dev)
    if rank == 0 and res is not None:
        print(json.dumps(res))
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
