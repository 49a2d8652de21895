"""Benchmark of the fused-attention hot path on GB300.

Default (N=1): the headline workload is Flash Attention prefill, B=4, Hq=Hkv=32,
Sq=Skv=2048, D=128, non-causal, bf16 inputs i.i.d. N(0,1) from the seeded generator.
One "step" is one prefill launch over that batch; `value` is TFLOP/s (4*B*H*Sq*Skv*D
per step).  The same run also measures, each with its own warm-up and timed loop:
the causal variant, the long-sequence prefills (S=8192, Hq=32/Hkv=8 D=128 and
Hq=64/Hkv=16 D=64, causal), batched Flash Decode (B=16, Hq=32, Hkv=8, lengths
U[4096,8192], 16 splits) and long-context Flash Decode (B=1, Hq=32, Hkv=8, Skv=131072,
model-chosen splits), reported under "workloads" with their own rooflines.

--impl reference times the fp64 CPU oracle (the reference arm) on host cores on a
bounded sample of the same workload and prints the same metric.

Multi-GPU (torchrun, one rank per GPU): every rank runs an independent replica of the
workload (the problems are independent; there is no data-path collective), timing is
bracketed by barriers and the max over ranks is taken; `value` counts all ranks' work.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import synth  # noqa: E402

METRIC = "attn fwd TFLOP/s & % of BF16 peak; decode KV GB/s & % of HBM BW (1 GB300)"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


# ------------------------------------------------------------------ environment
def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return {k: float(d[k]) for k in ("hbm_gbs", "bf16_tflops", "bf16_tflops_sustained")}, "measured"
    except Exception:
        return dict(FALLBACK_PEAKS), "fallback"


class ClockSampler:
    """Samples nvidia-smi clocks and throttle reasons while a timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap,clocks.mem")

    def __init__(self, device_index: int):
        self.dev = device_index
        self.proc = None
        self.lines = []
        self.t0 = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "100",
                 "-i", str(self.dev)], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.reader = threading.Thread(target=self._read, daemon=True)
            self.reader.start()
            time.sleep(0.3)
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.time(), line.strip()))

    def now(self):
        return time.time()

    def window(self, t0, t1):
        """Median SM/memory clock and throttle reasons seen between t0 and t1."""
        sms, maxes, mems, reasons = [], [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for t, line in list(self.lines):
            if not (t0 - 0.12 <= t <= t1 + 0.12):
                continue
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 10:
                continue
            try:
                sms.append(float(parts[1]))
                maxes.append(float(parts[2]))
                mems.append(float(parts[9]))
            except ValueError:
                continue
            for name, val in zip(names, parts[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        if not sms:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples in timed region"]}
        return {"sm_mhz": statistics.median(sms), "sm_max_mhz": max(maxes), "mem_mhz": statistics.median(mems),
                "samples": len(sms), "reasons": sorted(reasons)}

    def stop(self):
        if self.proc is None:
            return
        self.proc.terminate()
        try:
            self.proc.wait(timeout=2)
        except Exception:
            self.proc.kill()


# ------------------------------------------------------------------ workloads
# DRAM traffic (dram__bytes_read.sum + dram__bytes_write.sum) of one launch of the
# headline prefill kernel from an ncu capture of it, and the SHA-256 of the kernel
# sources it was taken from: the number is reported only while the sources are unchanged.
PROFILED_TRAFFIC_BYTES = 243.3e6
PROFILED_SOURCES_SHA256 = "41bf7a90c52cf9681ef9acb209e2175f44f8f01027f263dd1ad04d0645e58193"


def profiled_traffic():
    import hashlib
    h = hashlib.sha256()
    csrc = os.path.join(os.path.dirname(os.path.abspath(__file__)), "paper_2609_29219_gb300", "csrc")
    for f in ("attn_fwd.cu", "ptx.cuh", "kernels.h", "model.h"):
        with open(os.path.join(csrc, f), "rb") as fh:
            h.update(fh.read())
    return PROFILED_TRAFFIC_BYTES if h.hexdigest() == PROFILED_SOURCES_SHA256 else None


def headline_config(wl, world):
    """The `config` of the headline workload, the same object on both arms' lines."""
    return {"workload": wl.describe(), "B": 4, "Hq": 32, "Hkv": 32, "Sq": 2048, "Skv": 2048, "D": 128,
            "causal": False, "global_batch": 4 * world, "seq_len": 2048,
            "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
            "l2": "inputs larger than L2 (268 MB per step), 2 rotating input sets"}


def prefill_flops(B, Hq, Sq, Skv, D, causal):
    """Algorithmic FLOPs: 4*D per visible (query, key) pair (QK^T and PV, 2 FLOP per MAC)."""
    if not causal:
        pairs = Sq * Skv
    else:
        off = Skv - Sq
        pairs = sum(min(Skv, i + off + 1) for i in range(Sq))
    return 4.0 * B * Hq * D * pairs


class Prefill:
    def __init__(self, name, B, Hq, Hkv, S, D, causal, seed=0, sets=2):
        self.name, self.B, self.Hq, self.Hkv, self.S, self.D, self.causal = name, B, Hq, Hkv, S, D, causal
        self.seed, self.sets = seed, sets
        self.flops = prefill_flops(B, Hq, S, S, D, causal)
        # algorithmic HBM bytes: read Q, K, V once, write O and LSE
        self.bytes = 2 * (B * Hq * S * D * 2 + B * Hkv * S * D * 2) + B * Hq * S * 4
        self.unit = "TFLOP/s"

    def describe(self):
        return (f"prefill B={self.B} Hq={self.Hq} Hkv={self.Hkv} Sq=Skv={self.S} D={self.D} "
                f"{'causal' if self.causal else 'non-causal'}")

    def host_inputs(self, s):
        seed = self.seed + s
        return (synth.bf16_normal(seed, synth.STREAM_Q, (self.B, self.Hq, self.S, self.D)),
                synth.bf16_normal(seed, synth.STREAM_K, (self.B, self.Hkv, self.S, self.D)),
                synth.bf16_normal(seed, synth.STREAM_V, (self.B, self.Hkv, self.S, self.D)))

    def setup(self, torch, dev, loom):
        self.loom = loom
        self.inp = []
        for s in range(self.sets):
            q, k, v = (to_tensor(torch, x, dev) for x in self.host_inputs(s))
            o = torch.empty_like(q)
            lse = torch.empty((self.B, self.Hq, self.S), dtype=torch.float32, device=dev)
            self.inp.append((q, k, v, o, lse))

    def launches_per_step(self):
        return 1

    def step(self, i, stream):
        q, k, v, o, lse = self.inp[i % self.sets]
        self.loom.loom_attn_fwd(q, k, v, o, lse, causal=self.causal, stream=stream)

    def value(self, seconds_per_step):
        return self.flops / seconds_per_step / 1e12

    # end to end through the public API with host buffers
    def e2e_setup(self, torch, dev):
        """End-to-end steps through the public API: each step copies its inputs from
        pinned host memory, runs the kernel and copies O and LSE back.  Steps are
        pipelined over two device buffer sets, with host-to-device and device-to-host
        copies on their own streams, so that step i's kernel overlaps step i+1's input
        copies and step i-1's result copies."""
        q, k, v = self.host_inputs(0)
        pin = lambda a: to_host_tensor(torch, a).pin_memory()
        self.h_in = [pin(q), pin(k), pin(v)]
        self.h_o = [torch.empty(q.shape, dtype=torch.bfloat16).pin_memory() for _ in range(2)]
        self.h_lse = [torch.empty((self.B, self.Hq, self.S), dtype=torch.float32).pin_memory() for _ in range(2)]
        self.d_in2 = [[torch.empty(t.shape, dtype=t.dtype, device=dev) for t in self.h_in] for _ in range(2)]
        self.d_o2 = [torch.empty(q.shape, dtype=torch.bfloat16, device=dev) for _ in range(2)]
        self.d_lse2 = [torch.empty(self.h_lse[0].shape, dtype=torch.float32, device=dev) for _ in range(2)]
        self.s_h2d = torch.cuda.Stream(dev)
        self.s_d2h = torch.cuda.Stream(dev)
        self.ev_in = [torch.cuda.Event() for _ in range(2)]    # inputs of buffer set b landed
        self.ev_done = [torch.cuda.Event() for _ in range(2)]  # kernel on set b finished
        self.ev_out = [torch.cuda.Event() for _ in range(2)]   # results of set b copied back
        self.e2e_i = 0
        self.h2d = sum(t.numel() * t.element_size() for t in self.h_in)
        self.d2h = self.h_o[0].numel() * 2 + self.h_lse[0].numel() * 4
        # the single-step form below (tests, e2e of one call) uses buffer set 0
        self.d_in, self.d_o, self.d_lse = self.d_in2[0], self.d_o2[0], self.d_lse2[0]

    def e2e_step(self, stream):
        torch = self.torch
        i, b = self.e2e_i, self.e2e_i % 2
        self.e2e_i += 1
        if i >= 2:  # set b's previous kernel and result copies must be done with it
            self.s_h2d.wait_event(self.ev_done[b])
        with torch.cuda.stream(self.s_h2d):
            for d, h in zip(self.d_in2[b], self.h_in):
                d.copy_(h, non_blocking=True)
            self.ev_in[b].record(self.s_h2d)
        stream.wait_event(self.ev_in[b])
        if i >= 2:
            stream.wait_event(self.ev_out[b])
        self.loom.loom_attn_fwd(*self.d_in2[b], self.d_o2[b], self.d_lse2[b], causal=self.causal, stream=stream)
        self.ev_done[b].record(stream)
        self.s_d2h.wait_event(self.ev_done[b])
        with torch.cuda.stream(self.s_d2h):
            self.h_o[b].copy_(self.d_o2[b], non_blocking=True)
            self.h_lse[b].copy_(self.d_lse2[b], non_blocking=True)
            self.ev_out[b].record(self.s_d2h)

    def e2e_join(self, stream):
        """Make `stream` wait for every copy issued so far."""
        for b in range(2):
            stream.wait_event(self.ev_out[b])


class Decode:
    def __init__(self, name, B, Hq, Hkv, Skv, D, splits, lengths=None, seed=0, sets=2):
        self.name, self.B, self.Hq, self.Hkv, self.Skv, self.D = name, B, Hq, Hkv, Skv, D
        self.splits, self.seed, self.sets = splits, seed, sets
        self.lens = None if lengths is None else np.asarray(lengths, np.int32)
        total = int(self.lens.sum()) if self.lens is not None else B * Skv
        # algorithmic bytes: the K and V rows actually needed + q + o + lse
        self.bytes = 2 * Hkv * total * D * 2 + 2 * B * Hq * D * 2 + B * Hq * 4
        self.flops = 4.0 * Hq * total * D
        self.unit = "GB/s"

    def describe(self):
        ln = "lengths U[4096,8192]" if self.lens is not None else f"Skv={self.Skv}"
        return (f"decode B={self.B} Hq={self.Hq} Hkv={self.Hkv} Skv_max={self.Skv} D={self.D} {ln} "
                f"splits={self.splits or 'model'}")

    def host_inputs(self, s):
        seed = self.seed + s
        return (synth.bf16_normal(seed, synth.STREAM_Q, (self.B, self.Hq, 1, self.D)),
                synth.bf16_normal(seed, synth.STREAM_K, (self.B, self.Hkv, self.Skv, self.D)),
                synth.bf16_normal(seed, synth.STREAM_V, (self.B, self.Hkv, self.Skv, self.D)))

    def setup(self, torch, dev, loom):
        self.loom = loom
        self.inp = []
        self.sl = None if self.lens is None else torch.from_numpy(self.lens).to(dev)
        nbytes = loom.loom_attn_decode_workspace_bytes(self.B, self.Hq, self.Hkv, self.Skv, self.D, self.splits)
        self.ws = torch.empty(nbytes, dtype=torch.uint8, device=dev)
        self.used_splits = self.splits or loom.loom_attn_decode_num_splits(self.B, self.Hq, self.Hkv, self.Skv, self.D)
        for s in range(self.sets):
            q, k, v = (to_tensor(torch, x, dev) for x in self.host_inputs(s))
            o = torch.empty_like(q)
            lse = torch.empty((self.B, self.Hq), dtype=torch.float32, device=dev)
            self.inp.append((q, k, v, o, lse))

    def launches_per_step(self):
        return 2

    def step(self, i, stream):
        q, k, v, o, lse = self.inp[i % self.sets]
        self.loom.loom_attn_decode(q, k, v, self.sl, o, lse, self.ws, num_splits=self.splits, stream=stream)

    def value(self, seconds_per_step):
        return self.bytes / seconds_per_step / 1e9


class PagedDecode(Decode):
    """The batched decode over a paged cache [num_pages, page_size, Hkv, D]: each sequence's
    pages are dealt in a seeded shuffled order across the cache (a cache that has served
    many requests), so consecutive logical pages are scattered in HBM."""

    def __init__(self, name, B, Hq, Hkv, Skv, D, splits, page_size, lengths, seed=0, sets=2, layout="nhd",
                 in_order=False):
        super().__init__(name, B, Hq, Hkv, Skv, D, splits, lengths=lengths, seed=seed, sets=sets)
        self.P, self.layout, self.in_order = page_size, layout, in_order

    def describe(self):
        pages = "pages in order" if self.in_order else "pages shuffled"
        return super().describe().replace("decode ", f"paged decode ({self.layout}, {pages}) page_size={self.P} ", 1)

    def paged(self, k, v, s):
        B, Hkv, S, D, P = self.B, self.Hkv, self.Skv, self.D, self.P
        npg = S // P
        if self.in_order:  # page p of sequence b is cache page b * npg + p
            order = np.arange(B * npg, dtype=np.int32)
        else:
            order = np.random.default_rng(self.seed + s).permutation(B * npg).astype(np.int32)
        kc = np.empty((B * npg, P, Hkv, D), np.uint16)
        vc = np.empty_like(kc)
        kc[order] = k.reshape(B, Hkv, npg, P, D).transpose(0, 2, 3, 1, 4).reshape(B * npg, P, Hkv, D)
        vc[order] = v.reshape(B, Hkv, npg, P, D).transpose(0, 2, 3, 1, 4).reshape(B * npg, P, Hkv, D)
        if self.layout == "hnd":
            kc = np.ascontiguousarray(kc.transpose(0, 2, 1, 3))
            vc = np.ascontiguousarray(vc.transpose(0, 2, 1, 3))
        return kc, vc, order.reshape(B, npg)

    def setup(self, torch, dev, loom):
        self.loom = loom
        self.inp = []
        self.sl = torch.from_numpy(self.lens).to(dev)
        nbytes = loom.loom_attn_decode_workspace_bytes(self.B, self.Hq, self.Hkv, self.Skv, self.D, self.splits)
        self.ws = torch.empty(nbytes, dtype=torch.uint8, device=dev)
        self.used_splits = self.splits or loom.loom_attn_decode_num_splits(self.B, self.Hq, self.Hkv, self.Skv, self.D)
        for s in range(self.sets):
            q, k, v = self.host_inputs(s)
            kc, vc, table = self.paged(k, v, s)
            q = to_tensor(torch, q, dev)
            self.inp.append((q, to_tensor(torch, kc, dev), to_tensor(torch, vc, dev),
                             torch.from_numpy(np.ascontiguousarray(table)).to(dev), torch.empty_like(q),
                             torch.empty((self.B, self.Hq), dtype=torch.float32, device=dev)))

    def step(self, i, stream):
        q, kc, vc, table, o, lse = self.inp[i % self.sets]
        self.loom.loom_attn_decode_paged(q, kc, vc, table, self.sl, o, lse, self.ws, num_splits=self.splits,
                                         stream=stream, layout=self.layout)


class VarlenPrefill:
    """Prefill over a ragged batch packed [total, H, D]: seeded lengths U[lo, hi], causal
    (each sequence attends to itself), FLOPs = 4 D per visible (query, key) pair."""

    def __init__(self, name, B, Hq, Hkv, lo, hi, D, causal=True, seed=0, sets=2):
        self.name, self.B, self.Hq, self.Hkv, self.D, self.causal = name, B, Hq, Hkv, D, causal
        self.seed, self.sets, self.lo, self.hi = seed, sets, lo, hi
        self.lens = synth.decode_lengths(seed + 1, B, lo, hi).astype(np.int64)
        self.cu = np.concatenate([[0], np.cumsum(self.lens)]).astype(np.int32)
        self.total = int(self.cu[-1])
        self.flops = float(sum(prefill_flops(1, Hq, int(n), int(n), D, causal) for n in self.lens))
        self.bytes = 2 * (self.total * Hq * D * 2 + self.total * Hkv * D * 2) + self.total * Hq * 4
        self.unit = "TFLOP/s"

    def describe(self):
        return (f"varlen prefill B={self.B} lengths U[{self.lo},{self.hi}] (total {self.total} tokens) "
                f"Hq={self.Hq} Hkv={self.Hkv} D={self.D} {'causal' if self.causal else 'non-causal'}")

    def setup(self, torch, dev, loom):
        self.loom = loom
        self.inp = []
        self.cq = torch.from_numpy(self.cu).to(dev)
        self.maxq = int(self.lens.max())
        for s in range(self.sets):
            seed = self.seed + s
            q = to_tensor(torch, synth.bf16_normal(seed, synth.STREAM_Q, (self.total, self.Hq, self.D)), dev)
            k = to_tensor(torch, synth.bf16_normal(seed, synth.STREAM_K, (self.total, self.Hkv, self.D)), dev)
            v = to_tensor(torch, synth.bf16_normal(seed, synth.STREAM_V, (self.total, self.Hkv, self.D)), dev)
            self.inp.append((q, k, v, torch.empty_like(q),
                             torch.empty((self.Hq, self.total), dtype=torch.float32, device=dev)))

    def launches_per_step(self):
        return 1

    def step(self, i, stream):
        q, k, v, o, lse = self.inp[i % self.sets]
        self.loom.loom_attn_fwd_varlen(q, k, v, self.cq, self.cq, self.maxq, o, lse, causal=self.causal,
                                       stream=stream)

    def value(self, seconds_per_step):
        return self.flops / seconds_per_step / 1e12


class Gemm:
    """C = A B in bf16 with fp32 accumulation (the paper's GEMM, Sec. 4); A, B seeded N(0, 1)
    drawn on the device.  `cublas` times torch.matmul (cuBLAS) on the same buffers."""

    def __init__(self, name, M, N, K, seed=0, sets=2, cublas=False):
        self.name, self.M, self.N, self.K, self.seed, self.sets, self.cublas = name, M, N, K, seed, sets, cublas
        self.flops = 2.0 * M * N * K
        self.bytes = 2 * (M * K + K * N + M * N)
        self.unit = "TFLOP/s"

    def describe(self):
        return f"gemm M={self.M} N={self.N} K={self.K} bf16"

    def setup(self, torch, dev, loom):
        self.loom, self.torch = loom, torch
        g = torch.Generator(device=dev).manual_seed(self.seed)
        self.inp = []
        for _ in range(self.sets):
            a = torch.randn(self.M, self.K, generator=g, device=dev).to(torch.bfloat16)
            b = torch.randn(self.K, self.N, generator=g, device=dev).to(torch.bfloat16)
            self.inp.append((a, b, torch.empty(self.M, self.N, dtype=torch.bfloat16, device=dev)))

    def launches_per_step(self):
        return 1

    def step(self, i, stream):
        a, b, c = self.inp[i % self.sets]
        if self.cublas:
            self.torch.matmul(a, b, out=c)
        else:
            self.loom.loom_gemm_bf16(a, b, c, stream=stream)

    def value(self, seconds_per_step):
        return self.flops / seconds_per_step / 1e12


def to_tensor(torch, bits, dev):
    return to_host_tensor(torch, bits).to(dev)


def to_host_tensor(torch, bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16)


# ------------------------------------------------------------------ ranks
def make_collectives(torch, world, device):
    """The two collectives of the timed loops: a barrier around them and the maximum of a
    time over ranks (every rank runs one independent replica; rank 0 reports the job).
    One rank: no-ops.  `device` is where the reduction tensor lives (a GPU for NCCL, the
    CPU for gloo)."""
    if world <= 1:
        return (lambda: None), (lambda x: float(x))
    import torch.distributed as dist

    def barrier():
        dist.barrier()

    def reduce_max(x):
        t = torch.tensor([float(x)], device=device)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        return float(t.item())

    return barrier, reduce_max


def job_value(per_rank_value, world):
    """Whole-job throughput: every rank processes the same units per step (weak scaling),
    timed by the slowest rank, so the job's value is N times one rank's value at the
    maximum time."""
    return per_rank_value * world


# ------------------------------------------------------------------ timing
WARMUP_SECONDS = 1.0  # clocks ramp up slowly after host-side idle periods


def time_steps(torch, wl, steps, warmup, stream, barrier, per_launch_events=False, warm_s=WARMUP_SECONDS):
    """Warm up (at least `warmup` steps and `warm_s` seconds of back-to-back work), then
    time exactly `steps` steps with CUDA events on `stream`: one event before the first
    step and one after the last.  Events recorded around every step (per_launch_events)
    cost the steps themselves: they serialise the launches and cancel the programmatic
    overlap of one decode call's kernels with the next (measured 5.5 us per prefill step,
    8 us per decode step), so the timed loops record none, and a launch's duration is the
    loop's duration per step."""
    t0 = time.perf_counter()
    i = 0
    with torch.cuda.stream(stream):
        while i < warmup or time.perf_counter() - t0 < warm_s:
            for _ in range(max(1, warmup)):
                wl.step(i, stream)
                i += 1
            stream.synchronize()
    warmup = i
    torch.cuda.synchronize()
    barrier()
    torch.cuda.synchronize()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(steps)] if per_launch_events else []
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        t_start.record(stream)
        for i in range(steps):
            if evs:
                evs[i][0].record(stream)
            wl.step(warmup + i, stream)
            if evs:
                evs[i][1].record(stream)
        t_end.record(stream)
    torch.cuda.synchronize()
    barrier()
    torch.cuda.synchronize()
    total_ms = t_start.elapsed_time(t_end)
    launch_ms = [a.elapsed_time(b) for a, b in evs]
    return total_ms, launch_ms


def measure(torch, wl, steps, warmup, stream, barrier, world, reduce_max, peaks, clocks=None, warm_s=WARMUP_SECONDS):
    t_wall0 = time.time()
    total_ms, launch_ms = time_steps(torch, wl, steps, warmup, stream, barrier, warm_s=warm_s)
    t_wall1 = time.time()
    window = (t_wall1 - total_ms * 1e-3, t_wall1)  # the timed loop ends at the final sync
    del t_wall0
    total_ms = reduce_max(total_ms)
    ms_per_step = total_ms / steps
    value = job_value(wl.value(ms_per_step * 1e-3), world)
    # a launch's duration: the timed loop's duration per step (one launch per prefill
    # step, the split and merge launches per decode step), gaps between launches included
    avg_launch_ms = statistics.mean(launch_ms) if launch_ms else ms_per_step
    if wl.unit == "TFLOP/s":
        achieved = wl.flops / (avg_launch_ms * 1e-3) / 1e12
        roof = {"bound": "tensor", "achieved": round(achieved, 2), "peak": peaks["bf16_tflops"],
                "unit": "TFLOP/s", "frac": round(achieved / peaks["bf16_tflops"], 4)}
    else:
        achieved = wl.bytes / (avg_launch_ms * 1e-3) / 1e9
        roof = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "frac": round(achieved / peaks["hbm_gbs"], 4)}
    res = {"value": round(value, 3), "unit": wl.unit, "ms_per_step": round(ms_per_step, 5),
           "avg_launch_ms": round(avg_launch_ms, 5), "roofline": roof}
    if clocks is not None:
        res["clocks"] = clocks.window(*window)
    return res


def measure_e2e(torch, wl, steps, warmup, stream, barrier, reduce_max, world):
    wl.torch = torch
    wl.e2e_setup(torch, stream.device)
    with torch.cuda.stream(stream):
        for _ in range(warmup):
            wl.e2e_step(stream)
    torch.cuda.synchronize()
    barrier()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        a.record(stream)
        wl.s_h2d.wait_event(a)  # no copy of the timed steps starts before the start event
        for _ in range(steps):
            wl.e2e_step(stream)
        wl.e2e_join(stream)     # ... and the end event follows the last result copy
        b.record(stream)
    torch.cuda.synchronize()
    ms = reduce_max(a.elapsed_time(b)) / steps
    return {"value": round(job_value(wl.value(ms * 1e-3), world), 3), "unit": wl.unit,
            "h2d_bytes_per_step": int(wl.h2d), "d2h_bytes_per_step": int(wl.d2h),
            "ms_per_step": round(ms, 4)}


# ------------------------------------------------------------------ CPU oracle leg
def oracle_sample(wl, budget_s, threads=0):
    """Time the fp64 oracle on whole (b, h) heads of the prefill workload until the
    time budget is used; returns (TFLOP/s, heads done, seconds, threads)."""
    import oracle
    oracle.build()
    q, k, v = wl.host_inputs(0)
    heads_total = wl.B * wl.Hq
    done, flops, t0 = 0, 0.0, time.perf_counter()
    per_head = wl.flops / heads_total
    while done < heads_total and time.perf_counter() - t0 < budget_s:
        b, h = divmod(done, wl.Hq)
        rows = (np.arange(wl.S, dtype=np.int64) + (b * wl.Hq + h) * wl.S)
        oracle.attention(q, k, v, causal=wl.causal, rows=rows, nthreads=threads)
        done += 1
        flops += per_head
    dt = time.perf_counter() - t0
    return flops / dt / 1e12, done, dt, threads or (os.cpu_count() or 1)


# ------------------------------------------------------------------ main
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["loom", "reference"], default="loom")
    ap.add_argument("--quick", action="store_true", help="headline workload only")
    ap.add_argument("--only", default=None,
                    help="comma-separated subset (and order) of the extra workloads to run")
    ap.add_argument("--oracle-seconds", type=float, default=12.0)
    ap.add_argument("--sweep", choices=["decode", "model", "gemm", "ablation", "paged"], default=None,
                    help="decode: model-vs-measured sweep of the decode split count; model: the analytic "
                         "model's ranking and accuracy over prefill designs and shapes and decode split "
                         "counts and shapes; gemm: the BF16 GEMM over the shape grid {256, 2048, 16384}^3 "
                         "against cuBLAS, every tile width measured (one JSON line per point); ablation: "
                         "the block-size ablation, every compiled neighbour of the model's prefill ring "
                         "depth, decode stage plan and GEMM ring depth measured beside the model's choice")
    ap.add_argument("--prefill-design", type=int, default=0,
                    help="with --ncu-case: force this prefill design (1-4) instead of the model's choice")
    ap.add_argument("--ncu-case", default=None,
                    help="profiling run: set up this workload (tiny, tiny_causal, prefill, prefill_causal, "
                         "long_prefill_d128, long_prefill_d64, varlen_prefill, batched_decode, paged_decode_p16, paged_decode_p64, "
                         "paged_decode_hnd_p16, "
                         "long_decode, "
                         "gemm_4096, gemm_16k_256_16k, gemm_256_256_16k, gemm_8192, cublas_8192 (torch.matmul), "
                         "batched_decode_persistent, batched_decode_cluster4, "
                         "varlen_prefill_small), run --steps "
                         "launches, print nothing")
    args = ap.parse_args()
    world, rank, local = dist_env()
    if args.warmup < 3:
        args.warmup = 3

    headline = Prefill("prefill", 4, 32, 32, 2048, 128, causal=False)
    if args.impl == "reference":
        return run_reference(args, headline, world, rank)

    import torch
    import paper_2609_29219_gb300 as loom
    from paper_2609_29219_gb300 import build as libbuild
    if not os.path.exists(loom.library_path()):
        libbuild.build()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    barrier, reduce_max = make_collectives(torch, world, dev)

    peaks, peak_src = load_peaks()
    stream = torch.cuda.Stream(dev)
    if args.ncu_case:
        return run_ncu_case(torch, loom, dev, stream, args)
    if args.sweep == "decode":
        return run_decode_sweep(torch, loom, dev, stream, args, peaks)
    if args.sweep == "model":
        return run_model_sweep(torch, loom, dev, stream, args, peaks)
    if args.sweep == "gemm":
        return run_gemm_sweep(torch, loom, dev, stream, args, peaks)
    if args.sweep == "ablation":
        return run_ablation_sweep(torch, loom, dev, stream, args, peaks)
    if args.sweep == "paged":
        return run_paged_sweep(torch, loom, dev, stream, args)

    # headline: prefill non-causal, with clocks sampled during the timed loop
    headline.setup(torch, dev, loom)
    clocks = ClockSampler(local)
    clocks.start()
    res = measure(torch, headline, args.steps, args.warmup, stream, barrier, world, reduce_max, peaks, clocks)
    clk = res.pop("clocks", None)
    loom.loom_attn_check_error(stream)
    e2e = measure_e2e(torch, headline, max(5, min(args.steps, 50)), 3, stream, barrier, reduce_max, world)
    loom.loom_attn_check_error(stream)
    headline.inp = None

    workloads = {}
    if not args.quick or args.only:
        lens = synth.decode_lengths(0, 16, 4096, 8192)
        extra = [
            Prefill("prefill_causal", 4, 32, 32, 2048, 128, causal=True),
            Prefill("long_prefill_d128", 1, 32, 8, 8192, 128, causal=True),
            Prefill("long_prefill_d64", 1, 64, 16, 8192, 64, causal=True),
            VarlenPrefill("varlen_prefill", 16, 32, 8, 1024, 8192, 128, causal=True),
            Decode("batched_decode", 16, 32, 8, 8192, 128, splits=16, lengths=lens),
            PagedDecode("paged_decode_p16", 16, 32, 8, 8192, 128, splits=16, page_size=16, lengths=lens),
            PagedDecode("paged_decode_p64", 16, 32, 8, 8192, 128, splits=16, page_size=64, lengths=lens),
            PagedDecode("paged_decode_hnd_p16", 16, 32, 8, 8192, 128, splits=16, page_size=16, lengths=lens,
                        layout="hnd"),
            Decode("long_decode", 1, 32, 8, 131072, 128, splits=0),
        ]
        if args.only:
            by_name = {wl.name: wl for wl in extra}
            extra = [by_name[n] for n in args.only.split(",") if n]
        for wl in extra:
            wl.setup(torch, dev, loom)
            r = measure(torch, wl, max(10, args.steps // 2), args.warmup, stream, barrier, world, reduce_max, peaks,
                        clocks)
            loom.loom_attn_check_error(stream)
            r["workload"] = wl.describe()
            if isinstance(wl, Prefill) and wl.causal:
                # the FlashAttention convention counts half the non-causal FLOPs
                fa = 0.5 * prefill_flops(wl.B, wl.Hq, wl.S, wl.S, wl.D, False)
                r["value_fa_convention"] = round(r["value"] * fa / wl.flops, 3)
            if isinstance(wl, Decode):
                r["splits"] = wl.used_splits
                r["kv_bytes_per_step"] = int(wl.bytes)
                # overhead beside the algorithmic bytes: the partials written and read back
                r["workspace_bytes_per_step"] = int(2 * wl.B * wl.Hq * wl.used_splits * (wl.D + 1) * 4)
            r["gpu_launches"] = wl.launches_per_step() * max(10, args.steps // 2)
            workloads[wl.name] = r
            wl.inp = None
            torch.cuda.empty_cache()

    clocks.stop()
    cpu = None
    if rank == 0 and world == 1:
        tf, heads, dt, thr = oracle_sample(headline, args.oracle_seconds)
        cpu = {"value": round(tf, 6), "unit": "TFLOP/s", "cores": thr, "kind": "oracle",
               "sample": f"{heads} of {headline.B * headline.Hq} (b,h) heads x all {headline.S} query rows "
                         f"of the headline workload, fp64, {dt:.1f} s"}

    if rank == 0:
        roof = dict(res["roofline"])
        roof["traffic"] = profiled_traffic()
        roof["peak_source"] = f"{peak_src} (MEASURED_PEAKS.json bf16 burst)" if peak_src == "measured" else peak_src
        line = {
            "metric": METRIC,
            "value": res["value"],
            "unit": "TFLOP/s",
            "n_gpus": world,
            "steps": args.steps,
            "warmup": args.warmup,
            "ms_per_step": res["ms_per_step"],
            "higher_is_better": True,
            "scaling": "weak",
            "vs_baseline": None,
            "dtype": "bf16",
            "data": "synthetic (seeded splitmix64/Box-Muller N(0,1) rounded to bf16)",
            "config": headline_config(headline, world),
            "roofline": roof,
            "cpu_baseline": cpu,
            "e2e": e2e,
            "gpu_launches": args.steps * headline.launches_per_step(),
            "clocks": clk,
            "workloads": workloads,
            "summary": summary_line(res, clk, workloads),
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def summary_line(headline, headline_clocks, workloads):
    """One short string per workload (value, unit, roofline fraction, median SM clock,
    throttle reasons), kept last in the JSON line so that a reader of only its tail sees
    every configuration."""
    def one(r, clk):
        txt = f"{r['value']:.1f} {r['unit']} frac={r['roofline']['frac']:.3f}"
        if clk and clk.get("sm_mhz"):
            txt += f" sm={clk['sm_mhz']:.0f}MHz"
            if clk.get("reasons"):
                txt += " " + "+".join(clk["reasons"])
        if "splits" in r:
            txt += f" splits={r['splits']}"
        return txt

    out = {"prefill": one(headline, headline_clocks)}
    for name, r in workloads.items():
        out[name] = one(r, r.get("clocks"))
    return out


def run_decode_sweep(torch, loom, dev, stream, args, peaks):
    """Measured vs modeled Flash Decode time over split counts (the model's choice is the
    point marked "model": true)."""
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    lens = synth.decode_lengths(0, 16, 4096, 8192)
    cases = [
        (Decode("long_decode", 1, 32, 8, 131072, 128, splits=0), [8, 16, 19, 24, 32, 38, 48, 57, 64, 76, 96, 114, 152]),
        (Decode("batched_decode", 16, 32, 8, 8192, 128, splits=16, lengths=lens), [1, 2, 3, 4, 6, 8, 12, 16, 19, 24, 32]),
    ]
    G = 32 // 8
    for wl, splits in cases:
        wl.setup(torch, dev, loom)
        chosen = loom.loom_attn_decode_num_splits(wl.B, wl.Hq, wl.Hkv, wl.Skv, wl.D)
        chosen_form = loom.loom_attn_decode_form(wl.B, wl.Hq, wl.Hkv, wl.Skv, wl.D, 0)
        slots = loom.loom_decode_persistent_slots(wl.D, G)
        for sp in sorted(set(splits + [chosen])):
            wl.splits = sp
            nbytes = loom.loom_attn_decode_workspace_bytes(wl.B, wl.Hq, wl.Hkv, wl.Skv, wl.D, sp)
            wl.ws = torch.empty(nbytes, dtype=torch.uint8, device=dev)
            # split + merge (its split kernel on the tensor cores, then on the CUDA cores), the
            # persistent CUDA-core split kernel + merge, then the cluster form with every
            # power-of-two cluster size dividing sp
            for form, cs, tc in [(1, 0, 1), (1, 0, 0), (2, 0, 1)] + [(3, c, 1) for c in (2, 4, 8, 16) if sp % c == 0]:
                n_fit = loom.loom_decode_max_clusters(wl.D, G, cs) if cs else 0
                if cs and n_fit < 1:
                    continue
                loom.loom_debug_decode_form(form, cs)
                loom.loom_debug_decode_tensor_cores(tc)
                r = measure(torch, wl, max(10, args.steps // 4), args.warmup, stream, lambda: None, 1, float, peaks)
                loom.loom_attn_check_error(stream)
                loom.loom_debug_decode_tensor_cores(1)
                if form == 3:
                    model_us = loom.loom_model_decode_cluster_time_us(sp, cs, wl.B, wl.Hq, wl.Hkv, wl.Skv, wl.D, n_fit)
                elif form == 2:
                    model_us = loom.loom_model_decode_persistent_time_us(sp, wl.B, wl.Hq, wl.Hkv, wl.Skv, wl.D, slots)
                elif tc:
                    model_us = loom.loom_model_decode_tc_time_us(sp, wl.B, wl.Hq, wl.Hkv, wl.Skv, wl.D, sms)
                else:
                    model_us = loom.loom_model_decode_time_us(sp, wl.B, wl.Hq, wl.Hkv, wl.Skv, wl.D, sms)
                name = {1: "split+merge" if tc else "split+merge (CUDA cores)", 2: "persistent+merge",
                        3: f"cluster{cs}"}[form]
                print(json.dumps({"sweep": "decode", "workload": wl.describe(), "splits": sp, "form": name,
                                  "model_choice": sp == chosen and tc == 1 and (form, cs if form == 3 else 0) == chosen_form,
                                  "measured_us": round(r["ms_per_step"] * 1e3, 2),
                                  "model_us": round(model_us, 2), "GB/s": r["value"],
                                  "frac": r["roofline"]["frac"]}), flush=True)
            loom.loom_debug_decode_form(0)
        wl.inp = None
        torch.cuda.empty_cache()


def run_model_sweep(torch, loom, dev, stream, args, peaks):
    """The analytic model against measurement (the paper's ablations, restated for this
    path): for prefill shapes, every feasible design's modeled and measured time (does the
    model's top-1 design measure best?); for decode shapes with uniform lengths, the
    model's five best split counts, measured (ranking), with the modeled and measured
    throughput of the chosen point (accuracy)."""
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    steps = max(10, args.steps // 4)
    prefill = [(1, 32, 32, 1024, 128, False), (4, 32, 32, 2048, 128, False), (4, 32, 32, 2048, 128, True),
               (2, 32, 32, 4096, 128, False), (1, 32, 8, 8192, 128, True), (1, 16, 16, 16384, 128, False),
               (16, 16, 16, 512, 128, False), (4, 32, 32, 2048, 64, False), (1, 64, 16, 8192, 64, True),
               (2, 32, 32, 4096, 64, False)]
    for B, H, Hkv, S, D, causal in prefill:
        wl = Prefill("sweep", B, H, Hkv, S, D, causal=causal)
        wl.setup(torch, dev, loom)
        chosen = loom.loom_model_fwd_plan(D)["design"]
        for design in (1, 2, 3, 4):
            model_us = loom.loom_model_fwd_time_us_design(design, B, H, S, S, D, causal)
            if model_us < 0:
                continue
            loom.loom_debug_prefill_design(design)
            r = measure(torch, wl, steps, args.warmup, stream, lambda: None, 1, float, peaks)
            loom.loom_attn_check_error(stream)
            print(json.dumps({"sweep": "model", "kind": "prefill", "workload": wl.describe(), "design": design,
                              "model_choice": design == chosen, "measured_us": round(r["ms_per_step"] * 1e3, 2),
                              "model_us": round(model_us, 2), "measured_tflops": r["value"],
                              "model_tflops": round(wl.flops / (model_us * 1e-6) / 1e12, 1)}), flush=True)
        loom.loom_debug_prefill_design(0)
        wl.inp = None
        torch.cuda.empty_cache()
    decode = [(1, 32, 8, 131072, 128), (1, 32, 8, 32768, 128), (4, 32, 8, 16384, 128), (16, 32, 8, 8192, 128),
              (64, 32, 8, 2048, 128), (1, 64, 16, 65536, 64)]
    names = {1: "split+merge", 2: "persistent+merge", 3: "cluster"}
    for B, Hq, Hkv, Skv, D in decode:
        wl = Decode("sweep", B, Hq, Hkv, Skv, D, splits=0)
        wl.setup(torch, dev, loom)
        G = Hq // Hkv
        slots = loom.loom_decode_persistent_slots(D, G)
        fits = {cs: loom.loom_decode_max_clusters(D, G, cs) for cs in range(1, 17)}
        n = min(1024, (Skv + 63) // 64)
        cands = []  # (modeled us, form, splits, cluster size): Eq. 9's candidates over forms and split counts
        # the split + merge form's split kernel runs on the tensor cores for up to 32 query
        # heads per kv head
        tc = G <= 32
        split_merge = loom.loom_model_decode_tc_time_us if tc else loom.loom_model_decode_time_us
        for sp in range(1, n + 1):
            cands.append((split_merge(sp, B, Hq, Hkv, Skv, D, sms), 1, sp, 0))
            if slots > 0 and not tc:  # the CUDA-core persistent kernel, where the tensor-core one does not run
                cands.append((loom.loom_model_decode_persistent_time_us(sp, B, Hq, Hkv, Skv, D, slots), 2, sp, 0))
            for cs in range(1, min(16, sp) + 1):
                if sp % cs == 0 and fits[cs] > 0:
                    t = loom.loom_model_decode_cluster_time_us(sp, cs, B, Hq, Hkv, Skv, D, fits[cs])
                    if t > 0:
                        cands.append((t, 3, sp, cs))
        cands.sort()
        chosen_splits = loom.loom_attn_decode_num_splits(B, Hq, Hkv, Skv, D)
        chosen_form = loom.loom_attn_decode_form(B, Hq, Hkv, Skv, D, 0)
        for rank, (model_us, form, sp, cs) in enumerate(cands[:5]):
            wl.splits = sp
            nbytes = loom.loom_attn_decode_workspace_bytes(B, Hq, Hkv, Skv, D, sp)
            wl.ws = torch.empty(nbytes, dtype=torch.uint8, device=dev)
            loom.loom_debug_decode_form(form, cs)
            r = measure(torch, wl, steps, args.warmup, stream, lambda: None, 1, float, peaks)
            loom.loom_attn_check_error(stream)
            print(json.dumps({"sweep": "model", "kind": "decode", "workload": wl.describe(), "splits": sp,
                              "form": names[form] + (str(cs) if cs else ""), "model_rank": rank + 1,
                              "library_choice": sp == chosen_splits and (form, cs) == chosen_form,
                              "measured_us": round(r["ms_per_step"] * 1e3, 2),
                              "model_us": round(model_us, 2), "measured_gbs": r["value"],
                              "model_gbs": round(wl.bytes / (model_us * 1e-6) / 1e9, 1)}), flush=True)
        loom.loom_debug_decode_form(0)
        wl.inp = None
        torch.cuda.empty_cache()


def run_ablation_sweep(torch, loom, dev, stream, args, peaks):
    """The paper's block-size ablation restated for this path: around each constant the
    analytic model fixes (the prefill K/V ring depth, the decode stage plan, the GEMM ring
    depth), every neighbour that is compiled is timed on the benchmark workloads beside the
    model's choice (is the model's point locally best?)."""
    steps = max(10, args.steps // 4)

    def line(kind, wl, param, model, r):
        print(json.dumps({"sweep": "ablation", "kind": kind, "workload": wl.describe(), "param": param,
                          "model_choice": model, "measured_ms": round(r["ms_per_step"], 5), "value": r["value"],
                          "unit": r["unit"], "frac": r["roofline"]["frac"]}), flush=True)

    # prefill: ring depth of the two-tile design (BN = 128 keys is fixed by the softmax layout)
    lens = synth.decode_lengths(0, 16, 4096, 8192)
    prefill = [(Prefill("prefill", 4, 32, 32, 2048, 128, causal=False), (2, 3)),
               (Prefill("prefill_causal", 4, 32, 32, 2048, 128, causal=True), (2, 3)),
               (Prefill("long_prefill_d128", 1, 32, 8, 8192, 128, causal=True), (2, 3)),
               (Prefill("long_prefill_d64", 1, 64, 16, 8192, 64, causal=True), (3, 6, 9, 10)),
               (Prefill("prefill_d64", 4, 32, 32, 2048, 64, causal=False), (3, 6, 9, 10))]
    for wl, depths in prefill:
        wl.setup(torch, dev, loom)
        model_depth = loom.loom_model_fwd_plan_variant(wl.D, 2)["kv_slots"]
        for d in depths:
            assert loom.loom_debug_prefill_slots(wl.D, d)
            r = measure(torch, wl, steps, args.warmup, stream, lambda: None, 1, float, peaks)
            loom.loom_attn_check_error(stream)
            line("prefill_ring_depth", wl, {"kv_slots": d}, d == model_depth, r)
        loom.loom_debug_prefill_slots(wl.D, 0)
        wl.inp = None
        torch.cuda.empty_cache()

    # decode: keys per stage x ring stages x CTAs per SM of the split kernel (split + merge form)
    plans = [(64, 3, 2), (32, 2, 2), (32, 3, 2), (32, 4, 2), (64, 2, 2), (64, 4, 1), (128, 2, 1), (128, 3, 1)]
    loom.loom_debug_decode_form(1)  # the split + merge form, whose split kernel the plans change
    for wl in (Decode("batched_decode", 16, 32, 8, 8192, 128, splits=16, lengths=lens),
               Decode("long_decode", 1, 32, 8, 131072, 128, splits=0)):
        wl.setup(torch, dev, loom)
        for i, (t, st, c) in enumerate(plans):
            assert loom.loom_debug_decode_stage_plan(t, st, c)
            r = measure(torch, wl, steps, args.warmup, stream, lambda: None, 1, float, peaks)
            loom.loom_attn_check_error(stream)
            line("decode_stage_plan", wl, {"tokens": t, "stages": st, "ctas_per_sm": c}, i == 0, r)
        loom.loom_debug_decode_stage_plan(0)
        wl.inp = None
        torch.cuda.empty_cache()
    loom.loom_debug_decode_form(0)

    # GEMM: K-stage ring depth of the kernel the model picks (deeper rings do not fit)
    for (M, N, K), kernel, depths in [((8192, 8192, 8192), "pair", (5, 6)), ((16384, 16384, 16384), "pair", (5, 6)),
                                      ((4096, 4096, 4096), 256, (3, 4)), ((2048, 2048, 16384), 128, (5, 6))]:
        wl = Gemm("ablation", M, N, K)
        wl.setup(torch, dev, loom)
        if kernel == "pair":
            loom.loom_debug_gemm_cta_pair(1)
        else:
            loom.loom_debug_gemm_cta_pair(-1)
            loom.loom_debug_gemm_tile_n(kernel)
            loom.loom_debug_gemm_splits(1)
        for d in depths:
            loom.loom_debug_gemm_stages(d if d != max(depths) else 0)
            r = measure(torch, wl, max(10, min(steps, 200)), args.warmup, stream, lambda: None, 1, float, peaks,
                        warm_s=0.25)
            loom.loom_attn_check_error(stream)
            line("gemm_ring_depth", wl, {"kernel": kernel, "stages": d}, d == max(depths), r)
        loom.loom_debug_gemm_stages(0)
        loom.loom_debug_gemm_cta_pair(0)
        loom.loom_debug_gemm_tile_n(0)
        loom.loom_debug_gemm_splits(0)
        wl.inp = None
        torch.cuda.empty_cache()


def run_paged_sweep(torch, loom, dev, stream, args):
    """Paged decode against page placement: the batched decode over the contiguous cache
    and over paged caches (token- and head-major, page sizes 16 to 256) with each
    sequence's pages shuffled across the cache or in order, timed interleaved in shuffled
    rounds on one box (GB/s of the same algorithmic bytes)."""
    import random
    lens = synth.decode_lengths(0, 16, 4096, 8192)
    shape = (16, 32, 8, 8192, 128)
    wls = {"contiguous": Decode("batched_decode", *shape, splits=16, lengths=lens)}
    for layout, P in (("nhd", 16), ("hnd", 16), ("nhd", 64), ("hnd", 256)):
        for in_order in (False, True):
            key = f"{layout}_p{P}_{'in_order' if in_order else 'shuffled'}"
            wls[key] = PagedDecode("paged", *shape, splits=16, page_size=P, lengths=lens, layout=layout,
                                   in_order=in_order)
    for wl in wls.values():
        wl.sets = 1
        wl.setup(torch, dev, loom)
    nbytes = wls["contiguous"].bytes
    steps = max(20, min(args.steps, 200))
    res = {k: [] for k in wls}
    rng = random.Random(9)
    with torch.cuda.stream(stream):
        for _ in range(8):
            order = list(wls)
            rng.shuffle(order)
            for key in order:
                wl = wls[key]
                for i in range(max(3, args.warmup)):
                    wl.step(i, stream)
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                for i in range(steps):
                    wl.step(i, stream)
                e1.record(stream)
                e1.synchronize()
                res[key].append(nbytes * steps / (e0.elapsed_time(e1) * 1e-3) / 1e9)
    loom.loom_attn_check_error(stream)
    for key, v in res.items():
        print(json.dumps({"sweep": "paged", "cache": key, "workload": wls[key].describe(),
                          "gbs_median": round(statistics.median(v), 1), "rounds": len(v)}), flush=True)


GEMM_DIMS = (256, 2048, 16384)


def run_gemm_sweep(torch, loom, dev, stream, args, peaks):
    """The BF16 GEMM over the paper's shape range (every M, N, K in {256, 2048, 16384}):
    cuBLAS (torch.matmul); this library with the model's choice; CTA-pair tiles; every tile
    width with single-CTA persistent tiles (S = 1); and, at the model's single-CTA tile
    width, every split count that leaves each CTA two K stages or more (does the model's
    choice measure best?).  All on the same buffers and stream."""
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    for M in GEMM_DIMS:
        for N in GEMM_DIMS:
            for K in GEMM_DIMS:
                wl = Gemm("sweep", M, N, K)
                wl.setup(torch, dev, loom)
                steps = int(min(500, max(10, 0.05 / (wl.flops / 1.5e15))))
                bn, sp = loom.loom_gemm_tile_n(M, N, K), loom.loom_gemm_splits(M, N, K)
                pair = loom.loom_gemm_cta_pair(M, N, K)
                row = {"sweep": "gemm", "workload": wl.describe(), "model_tile_n": bn, "model_splits": sp,
                       "model_cta_pair": pair,
                       "model_us": round(loom.loom_model_gemm_time_us(M, N, K, 512 if pair else bn, sp, sms), 2)}

                def timed():
                    r = measure(torch, wl, steps, args.warmup, stream, lambda: None, 1, float, peaks, warm_s=0.25)
                    loom.loom_attn_check_error(stream)
                    return r["value"]

                # the library's choice first: the GPU's clocks recover slowly after a long
                # cuBLAS run, which would bias whatever is timed right after it
                wl.cublas = False
                row["loom_tflops"] = timed()
                c = wl.inp[0][2].float()
                wl.cublas = True
                row["cublas_tflops"] = timed()
                ref = wl.inp[0][2].float()
                wl.cublas = False
                row["max_rel_diff_vs_cublas"] = float(f"{(c - ref).abs().max().item() / max(ref.abs().max().item(), 1e-30):.3g}")
                loom.loom_debug_gemm_cta_pair(1)
                row["pair_tflops"] = timed()
                loom.loom_debug_gemm_cta_pair(-1)
                for t in (64, 128, 192, 256):
                    loom.loom_debug_gemm_tile_n(t)
                    loom.loom_debug_gemm_splits(1)
                    row[f"bn{t}_s1_tflops"] = timed()
                loom.loom_debug_gemm_tile_n(0)
                loom.loom_debug_gemm_splits(0)
                sbn = loom.loom_gemm_tile_n(M, N, K)  # the model's single-CTA width (pairs forbidden)
                loom.loom_debug_gemm_tile_n(sbn)
                for s_ in (2, 4, 8, 16):
                    if (K + 63) // 64 < 2 * s_:
                        break
                    loom.loom_debug_gemm_splits(s_)
                    row[f"bn{sbn}_s{s_}_tflops"] = timed()
                loom.loom_debug_gemm_tile_n(0)
                loom.loom_debug_gemm_splits(0)
                loom.loom_debug_gemm_cta_pair(0)
                row["vs_cublas"] = round(row["loom_tflops"] / row["cublas_tflops"], 3)
                row["frac_of_peak"] = round(row["loom_tflops"] / peaks["bf16_tflops"], 4)
                print(json.dumps(row), flush=True)
                wl.inp = None
                del ref, c
                torch.cuda.empty_cache()


def all_workloads():
    lens = synth.decode_lengths(0, 16, 4096, 8192)
    return [Prefill("tiny", 1, 2, 2, 128, 64, causal=False),
            Prefill("tiny_causal", 1, 2, 2, 128, 64, causal=True),
            Prefill("prefill", 4, 32, 32, 2048, 128, causal=False),
            Prefill("prefill_causal", 4, 32, 32, 2048, 128, causal=True),
            Prefill("long_prefill_d128", 1, 32, 8, 8192, 128, causal=True),
            Prefill("long_prefill_d64", 1, 64, 16, 8192, 64, causal=True),
            VarlenPrefill("varlen_prefill", 16, 32, 8, 1024, 8192, 128, causal=True),
            Decode("batched_decode", 16, 32, 8, 8192, 128, splits=16, lengths=lens),
            PagedDecode("paged_decode_p16", 16, 32, 8, 8192, 128, splits=16, page_size=16, lengths=lens),
            PagedDecode("paged_decode_p64", 16, 32, 8, 8192, 128, splits=16, page_size=64, lengths=lens),
            PagedDecode("paged_decode_hnd_p16", 16, 32, 8, 8192, 128, splits=16, page_size=16, lengths=lens,
                        layout="hnd"),
            Decode("long_decode", 1, 32, 8, 131072, 128, splits=0)]


def run_ncu_case(torch, loom, dev, stream, args):
    """A few launches of one workload and nothing else, for small ncu captures."""
    cases = {w.name: w for w in all_workloads()}
    cases["gemm_4096"] = Gemm("gemm_4096", 4096, 4096, 4096)
    cases["gemm_16k_256_16k"] = Gemm("gemm_16k_256_16k", 16384, 256, 16384)
    cases["gemm_256_256_16k"] = Gemm("gemm_256_256_16k", 256, 256, 16384)
    cases["gemm_8192"] = Gemm("gemm_8192", 8192, 8192, 8192)
    cases["cublas_8192"] = Gemm("cublas_8192", 8192, 8192, 8192, cublas=True)
    cases["varlen_prefill_small"] = VarlenPrefill("varlen_prefill_small", 8, 32, 8, 512, 2048, 128, causal=True)
    cases["prefill_d64_small"] = Prefill("prefill_d64_small", 1, 16, 4, 8192, 64, causal=True)
    cases["batched_decode_persistent"] = Decode("batched_decode", 16, 32, 8, 8192, 128, splits=16,
                                             lengths=synth.decode_lengths(0, 16, 4096, 8192))
    cases["batched_decode_cluster4"] = Decode("batched_decode", 16, 32, 8, 8192, 128, splits=16,
                                           lengths=synth.decode_lengths(0, 16, 4096, 8192))
    wl = cases[args.ncu_case]
    if args.prefill_design:
        loom.loom_debug_prefill_design(args.prefill_design)
    if args.ncu_case == "batched_decode_persistent":
        loom.loom_debug_decode_form(2)
    if args.ncu_case == "batched_decode_cluster4":
        loom.loom_debug_decode_form(3, 4)  # the single-kernel form, clusters of 4 CTAs
    wl.sets = 1  # one input set: the smallest device footprint for a capture
    wl.setup(torch, dev, loom)
    with torch.cuda.stream(stream):
        for i in range(max(1, args.steps)):
            wl.step(i, stream)
    torch.cuda.synchronize()
    loom.loom_attn_check_error(stream)


def run_reference(args, wl, world, rank):
    """Reference arm: the fp64 oracle on host cores; each step is a bounded sample of
    the headline workload (512 query rows of one (b, h) head, heads rotating)."""
    if rank != 0:
        return
    import oracle
    oracle.build()
    q, k, v = wl.host_inputs(0)
    rows_per_step = 512
    heads = wl.B * wl.Hq
    per_row = wl.flops / (heads * wl.S)  # non-causal: every row costs the same

    def step(i):
        head = i % heads
        r0 = (i // heads * rows_per_step) % wl.S
        rows = np.arange(r0, r0 + rows_per_step, dtype=np.int64) % wl.S + head * wl.S
        oracle.attention(q, k, v, causal=wl.causal, rows=rows)

    for i in range(args.warmup):
        step(i)
    t0 = time.perf_counter()
    for i in range(args.steps):
        step(args.warmup + i)
    dt = time.perf_counter() - t0
    ms = dt * 1e3 / args.steps
    value = rows_per_step * per_row / (ms * 1e-3) / 1e12
    cores = os.cpu_count() or 1
    line = {
        "impl": "reference",
        "metric": METRIC, "value": round(value, 6), "unit": "TFLOP/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded splitmix64/Box-Muller N(0,1) rounded to bf16)",
        "config": headline_config(wl, world),
        "cpu_baseline": {"value": round(value, 6), "unit": "TFLOP/s", "cores": cores, "kind": "oracle",
                         "sample": f"{rows_per_step} query rows of one (b,h) head per step (fp64 oracle, "
                                   f"{cores} threads)"},
        "e2e": {"value": round(value, 6), "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
