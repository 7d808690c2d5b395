#!/usr/bin/env python3
"""Benchmark of the thin-key attention hot path on GB300.

Headline (one JSON line on stdout): decode KV GB/s of the Mistral-7B-shaped
GQA decode (B=16, H_q=32, H_kv=8, r=32, d_v=128, every context 4096 tokens).
One step = one pass of the decode path over the batch: tk_kv_append of the
new token of every sequence (written at position 4095, so the context stays
4096) followed by tk_attn_decode (split-KV partials and their merge, one
launch).  The line also carries tokens/s, the roofline of the decode kernel,
the end-to-end number through host buffers, the oracle's CPU throughput,
SM clocks sampled during the timed region, and the other workloads
(causal prefill TFLOP/s, paged long-context decode, int8-key decode with
its r sweep, the GPT-2-small layer).

Timing: CUDA graphs of the step sequence are replayed between two CUDA
events on the launching stream; W untimed warm-up steps first.  The decode
workload rotates over several cache copies whose total exceeds 4x L2, so
no step reads cache lines left by the previous one.

    python bench.py [--gpus N --steps K --warmup W] [--impl reference]
"""

from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "decode KV GB/s (% HBM peak), tokens/s; prefill TFLOP/s (% bf16 peak), 1 GB300"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def log(*a):
    print(*a, file=sys.stderr, flush=True)


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        d = json.load(open(p))
        return {k: float(d[k]) for k in FALLBACK_PEAKS}, "measured"
    except Exception:
        return dict(FALLBACK_PEAKS), "fallback"


def source_hash(*names):
    h = hashlib.sha256()
    for n in names:
        h.update(open(os.path.join(ROOT, "paper_2603_04427_gb300", "csrc", n), "rb").read())
    return h.hexdigest()[:16]


def recorded_traffic(kernel: str, workload: str, src_hash: str):
    """DRAM bytes per launch from a committed ncu capture, if the kernel is unchanged since."""
    try:
        d = json.load(open(os.path.join(ROOT, "profiles", "dram_traffic.json")))
        e = d[kernel][workload]
        return e["bytes_per_launch"] if e.get("source_hash") == src_hash else None
    except Exception:
        return None


# ----------------------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons while it runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,utilization.gpu,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        time.sleep(0.2)

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        rows = []
        for line in open(self.path):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) >= 9:
                rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None

        sm = [num(r[1]) for r in rows if num(r[1]) is not None]
        util = [num(r[4]) or 0.0 for r in rows]
        loaded = [num(r[1]) for r, u in zip(rows, util) if u >= 50 and num(r[1]) is not None]
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if v.strip() == "Active"})
        return {"sm_mhz": statistics.median(loaded or sm), "sm_max_mhz": max(num(r[2]) or 0 for r in rows),
                "reasons": reasons, "samples": len(rows), "samples_under_load": len(loaded)}


# ----------------------------------------------------------------------------- GPU side

def _l2_bytes(torch):
    try:
        return int(torch.cuda.get_device_properties(torch.cuda.current_device()).L2_cache_size)
    except Exception:
        return 129 * 2 ** 20


class DecodeRig:
    """Caches, inputs and pre-marshalled C-ABI arguments for one decode workload.

    Each copy is a complete cache plus its query / new-token / output / workspace
    buffers; steps rotate over the copies.
    """

    def __init__(self, w, device, copies=None, k_fmt=None, r=None):
        import torch

        from paper_2603_04427_gb300 import binding as tb
        from paper_2603_04427_gb300 import inputs
        self.tb, self.torch = tb, torch
        self.w = w
        self.r = r or w.r
        # key storage: "bf16", "int8" or "int4" (two codes per byte)
        self.k_fmt = ("int8" if w.k_int8 else "bf16") if k_fmt is None else k_fmt
        self.k_int8 = self.k_fmt == "int8"
        self.k_int4 = self.k_fmt == "int4"
        B, hq, hkv, dv = w.batch, w.h_q, w.h_kv, w.d_v
        if w.seq_range:
            self.lens = inputs.uniform_lengths(B, w.seq_range[0], w.seq_range[1], seed=w.seed)
        else:
            self.lens = [w.seq] * B
        self.max_len = max(self.lens)
        from paper_2603_04427_gb300 import cost_model as cm
        k_row = {"bf16": 2 * self.r, "int8": self.r, "int4": self.r // 2}[self.k_fmt]
        self.kv_bytes = cm.decode_kv_bytes(self.lens, hkv, k_row, dv, k_bytes=1,
                                           k_scale_bytes=0 if self.k_fmt == "bf16" else 4)
        self.io_bytes = cm.decode_io_bytes(B, hq, self.r, dv, out_bytes=4)
        per_copy = self.kv_bytes
        if copies is None:
            copies = max(1, min(8, math.ceil(4 * _l2_bytes(torch) / per_copy)))
        self.copies = []
        seq_app = torch.tensor([n - 1 for n in self.lens], dtype=torch.int32, device=device)
        seq_dec = torch.tensor(self.lens, dtype=torch.int32, device=device)
        for c in range(copies):
            seed = w.seed * 100 + c * 10
            if w.page_size:
                table, n_pages = inputs.paged_layout(self.lens, w.page_size, seed=seed)
                cache = tb.ThinKeyCache.allocate(B, hq, hkv, self.r, dv, page_size=w.page_size,
                                                 num_pages=n_pages, page_table=table,
                                                 k_int8=self.k_int8, k_int4=self.k_int4,
                                                 device=device)
                self._fill_paged(cache, seed, device)
            else:
                cap = (self.max_len + 15) // 16 * 16
                cache = tb.ThinKeyCache.allocate(B, hq, hkv, self.r, dv, capacity=cap,
                                                 k_int8=self.k_int8, k_int4=self.k_int4,
                                                 device=device)
                T = self.max_len
                kn = inputs.normal_bf16((B, hkv, T, self.r), seed + 1, device=device)
                vn = inputs.normal_bf16((B, hkv, T, dv), seed + 2, device=device)
                tb.tk_kv_append(cache, kn, vn, torch.zeros(B, dtype=torch.int32, device=device))
                del kn, vn
            # the step's inputs (query, new key, new value) in one buffer, so the
            # end-to-end leg moves them with one host-to-device copy
            nq, nk, nv = B * hq * self.r, B * hkv * self.r, B * hkv * dv
            io = torch.empty(nq + nk + nv, dtype=torch.bfloat16, device=device)
            q, k1, v1 = io[:nq].view(B, hq, self.r), io[nq:nq + nk].view(B, hkv, 1, self.r), \
                io[nq + nk:].view(B, hkv, 1, dv)
            q.copy_(inputs.normal_bf16((B, hq, self.r), seed + 3, device=device))
            k1.copy_(inputs.normal_bf16((B, hkv, 1, self.r), seed + 4, device=device))
            v1.copy_(inputs.normal_bf16((B, hkv, 1, dv), seed + 5, device=device))
            out = torch.empty(B, hq, dv, dtype=torch.float32, device=device)
            ws = tb.decode_workspace(cache.desc, self.max_len, device=device)
            self.copies.append(dict(cache=cache, io=io, q=q, k1=k1, v1=v1, out=out, ws=ws,
                                    seq_app=seq_app, seq_dec=seq_dec))
        torch.cuda.synchronize()
        if tb.tk_get_device_error() != 0:
            raise RuntimeError("device error while building the cache")

    def _fill_paged(self, cache, seed, device):
        from paper_2603_04427_gb300 import inputs
        torch = self.torch
        if self.k_fmt != "bf16":
            raise NotImplementedError("paged quantised-key rig is not used by the benchmark")
        cache.k.copy_(inputs.normal_bf16(cache.k.shape, seed + 1, device=device))
        cache.v.copy_(inputs.normal_bf16(cache.v.shape, seed + 2, device=device))

    def step(self, i, mode="fused"):
        """One decode step on copy i: "fused" = tk_attn_decode_append (one launch),
        "append" = tk_kv_append + tk_attn_decode, "decode" = tk_attn_decode alone."""
        c = self.copies[i % len(self.copies)]
        if mode == "fused":
            cache = c["cache"]
            B, hkv = cache.desc.batch, cache.desc.h_kv
            self.tb.tk_attn_decode_append(cache, c["q"], c["k1"].view(B, hkv, -1),
                                          c["v1"].view(B, hkv, -1), c["seq_app"], self.max_len,
                                          c["out"], c["ws"])
            return
        if mode == "append":
            self.tb.tk_kv_append(c["cache"], c["k1"], c["v1"], c["seq_app"])
        self.tb.tk_attn_decode(c["cache"], c["q"], c["seq_dec"], self.max_len, c["out"], c["ws"])


def graph_time(torch, enqueue, steps, warmup, max_graph=256, min_seconds=0.0, info=None):
    """Seconds for exactly `steps` calls of enqueue(i), replayed from CUDA graphs.

    One block = the `steps` calls between two CUDA events on the launching
    stream.  With min_seconds > 0 blocks are replayed back to back until that
    much device time has passed, and the median block is returned (so that a
    short block is not decided by one replay, and clock samplers see load);
    `info` then receives the block count and the device time spanned."""
    stream = torch.cuda.Stream()
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        for i in range(warmup):
            enqueue(i)
    torch.cuda.synchronize()
    G = max(1, min(steps, max_graph))
    graphs = {}

    def graph_of(n):
        if n not in graphs:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                for i in range(n):
                    enqueue(i)
            graphs[n] = g
        return graphs[n]

    full, rem = divmod(steps, G)
    g_full = graph_of(G) if full else None
    g_rem = graph_of(rem) if rem else None

    def block():
        if g_full is not None:
            for _ in range(full):
                g_full.replay()
        if g_rem is not None:
            g_rem.replay()

    with torch.cuda.stream(stream):   # one untimed replay uploads the graphs
        block()
    torch.cuda.synchronize()
    times = []
    spent = 0.0
    while True:
        # a batch of blocks, each between its own pair of events
        n_blk = 1 if not times else max(1, min(512, int(len(times) * (min_seconds - spent) / spent) + 1))
        evs = [torch.cuda.Event(enable_timing=True) for _ in range(n_blk + 1)]
        with torch.cuda.stream(stream):
            evs[0].record(stream)
            for j in range(n_blk):
                block()
                evs[j + 1].record(stream)
        evs[-1].synchronize()
        new = [evs[j].elapsed_time(evs[j + 1]) / 1e3 for j in range(n_blk)]
        times += new
        spent += sum(new)
        if spent >= min_seconds:
            break
    if info is not None:
        info.update(blocks=len(times), timed_region_s=spent)
    return statistics.median(times)


def measure_decode(rig, steps, warmup, mode="fused", min_seconds=0.0, info=None):
    torch = rig.torch
    sec = graph_time(torch, lambda i: rig.step(i, mode), steps, warmup, min_seconds=min_seconds,
                     info=info)
    return sec / steps


def measure_decode_e2e(rig, steps, graph=True):
    """Through host buffers and the public API: per step the step's query, new
    key and new value come from one page-locked host buffer (tk_copy_async,
    issued with the fused append + decode as one call prepared once, as a
    serving loop with fixed buffers makes it; with graph=True the two are
    recorded once as a CUDA graph and each step is one tk_graph_launch), the
    kernel writes the output straight into a page-locked host buffer
    (zero-copy), and the host synchronises before the next step."""
    torch = rig.torch
    tb = rig.tb
    hio = [c["io"].cpu().pin_memory() for c in rig.copies]
    ho = torch.empty(rig.copies[0]["out"].shape, dtype=torch.float32).pin_memory()
    stream = torch.cuda.Stream()
    calls = []
    for c, h in zip(rig.copies, hio):
        cache = c["cache"]
        B, hkv = cache.desc.batch, cache.desc.h_kv
        calls.append(tb.prepare_decode_append(cache, c["q"], c["k1"].view(B, hkv, -1),
                                              c["v1"].view(B, hkv, -1), c["seq_app"], rig.max_len,
                                              ho, c["ws"], stream=stream, copy_in=(c["io"], h),
                                              graph=graph))
    n = max(1, steps)
    for i in range(min(n, 20)):  # warm-up
        calls[i % len(calls)]()
        stream.synchronize()
    t0 = time.perf_counter()
    for i in range(n):
        calls[i % len(calls)]()
        stream.synchronize()
    dt = (time.perf_counter() - t0) / n
    if not torch.isfinite(ho).all():
        raise RuntimeError("end-to-end decode produced a non-finite output")
    h2d = hio[0].numel() * 2
    d2h = ho.numel() * 4
    return dt, h2d, d2h


def measure_prefill(w, iters, device, torch):
    """Causal prefill, bf16 output, rotating input copies (> 4x L2 in total)."""
    from paper_2603_04427_gb300 import binding as tb
    from paper_2603_04427_gb300 import cost_model as cm
    from paper_2603_04427_gb300 import inputs
    B, hq, hkv, S, r, dv = w.batch, w.h_q, w.h_kv, w.seq, w.r, w.d_v
    per = (B * hq * S * r + B * hkv * S * (r + dv) + B * hq * S * dv) * 2
    copies = max(1, min(4, math.ceil(4 * _l2_bytes(torch) / per)))
    sets = []
    for c in range(copies):
        s = w.seed * 100 + c * 10
        sets.append((inputs.normal_bf16((B, hq, S, r), s + 1, device=device),
                     inputs.normal_bf16((B, hkv, S, r), s + 2, device=device),
                     inputs.normal_bf16((B, hkv, S, dv), s + 3, device=device),
                     torch.empty(B, hq, S, dv, dtype=torch.bfloat16, device=device)))
    try:
        q, k, v, o = sets[0]
        tb.tk_attn_prefill(q, k, v, o)
    except tb.TkError as e:
        if e.status == tb.TK_ERR_UNSUPPORTED:
            return {"status": "unsupported"}
        raise

    def enq(i):
        q, k, v, o = sets[i % len(sets)]
        tb.tk_attn_prefill(q, k, v, o)

    sec = graph_time(torch, enq, iters, 3, max_graph=16, min_seconds=0.5) / iters
    flops = cm.prefill_flops(B, hq, S, r, dv, causal=True)
    return {"ms": sec * 1e3, "tflops": flops / sec / 1e12, "flops_per_launch": flops}


def measure_chunked_prefill(w, iters, device, torch, k_fmt="bf16"):
    """A prompt chunk of w.seq tokens after w.cached cached ones: tk_attn_prefill_cached
    (append of the chunk, for int8 / int4 keys the widening of the context's keys into
    the workspace, attention over the cache), bf16 output; keys stored as bf16, int8 or
    int4.  The append launch is also timed on its own."""
    from paper_2603_04427_gb300 import binding as tb
    from paper_2603_04427_gb300 import cost_model as cm
    from paper_2603_04427_gb300 import inputs
    B, hq, hkv, S, r, dv, L0 = w.batch, w.h_q, w.h_kv, w.seq, w.r, w.d_v, w.cached
    cache = tb.ThinKeyCache.allocate(B, hq, hkv, r, dv, capacity=L0 + S, device=device,
                                     k_int8=k_fmt == "int8", k_int4=k_fmt == "int4")
    zero = torch.zeros(B, dtype=torch.int32, device=device)
    tb.tk_kv_append(cache, inputs.normal_bf16((B, hkv, L0, r), w.seed + 1, device=device),
                    inputs.normal_bf16((B, hkv, L0, dv), w.seed + 2, device=device), zero)
    q = inputs.normal_bf16((B, hq, S, r), w.seed + 3, device=device)
    kn = inputs.normal_bf16((B, hkv, S, r), w.seed + 4, device=device)
    vn = inputs.normal_bf16((B, hkv, S, dv), w.seed + 5, device=device)
    out = torch.empty(B, hq, S, dv, dtype=torch.bfloat16, device=device)
    sl = torch.full((B,), L0, dtype=torch.int32, device=device)
    ws = tb.prefill_cached_workspace(cache, L0 + S)

    def enq(_):  # the same chunk re-appended at the same positions every time
        tb.tk_attn_prefill_cached(cache, q, kn, vn, sl, L0 + S, out, workspace=ws)

    def enq_append(_):
        tb.tk_kv_append(cache, kn, vn, sl)

    sec = graph_time(torch, enq, iters, 3, max_graph=16, min_seconds=0.3) / iters
    sec_app = graph_time(torch, enq_append, iters, 3, max_graph=16, min_seconds=0.1) / iters
    flops = cm.prefill_flops(B, hq, S, r, dv, cached=L0)
    return {"ms": sec * 1e3, "tflops": flops / sec / 1e12, "flops_per_call": flops,
            "cached": L0, "launches": 2 if k_fmt == "bf16" else 3, "append_ms": sec_app * 1e3,
            "k_dtype": k_fmt}


def measure_backward(w, iters, device, torch):
    """Training backward of the causal prefill shape (tk_attn_backward: the D / dQ-zeroing
    pass and the gradient kernel), from a tk_attn_forward of the same inputs."""
    from paper_2603_04427_gb300 import binding as tb
    from paper_2603_04427_gb300 import cost_model as cm
    from paper_2603_04427_gb300 import inputs
    B, hq, hkv, S, r, dv = w.batch, w.h_q, w.h_kv, w.seq, w.r, w.d_v
    q = inputs.normal_bf16((B, hq, S, r), w.seed + 1, device=device)
    k = inputs.normal_bf16((B, hkv, S, r), w.seed + 2, device=device)
    v = inputs.normal_bf16((B, hkv, S, dv), w.seed + 3, device=device)
    do = inputs.normal_bf16((B, hq, S, dv), w.seed + 4, device=device)
    out = torch.empty(B, hq, S, dv, dtype=torch.bfloat16, device=device)
    lse = torch.empty(B, hq, S, dtype=torch.float32, device=device)
    tb.tk_attn_forward(q, k, v, out, lse)
    dq = torch.empty(B, hq, S, r, dtype=torch.float32, device=device)
    dk = torch.empty(B, hkv, S, r, dtype=torch.float32, device=device)
    dvv = torch.empty(B, hkv, S, dv, dtype=torch.float32, device=device)
    ws = torch.empty(int(tb.load_library().tk_backward_workspace_size(B, hq, S)), dtype=torch.uint8,
                     device=device)

    def enq(_):
        tb.tk_attn_backward(q, k, v, out, do, lse, dq, dk, dvv, ws)

    sec = graph_time(torch, enq, iters, 3, max_graph=8, min_seconds=0.3) / iters
    pairs = cm.causal_pairs(S) * B * hq
    flops = pairs * 2 * (3 * r + 2 * dv)   # S^T, dP^T, dV, dK, dQ products
    return {"ms": sec * 1e3, "tflops": flops / sec / 1e12, "flops_per_call": flops, "launches": 2}


def measure_gpt2_layer(w, iters, device, torch):
    """GPT-2-small layer: causal prefill of S tokens (fp32 out), append of the
    prompt's keys/values, then `decode_steps` x (append 1 token + decode)."""
    from paper_2603_04427_gb300 import binding as tb
    from paper_2603_04427_gb300 import cost_model as cm
    from paper_2603_04427_gb300 import inputs
    B, H, r, dv, S, T = w.batch, w.h_q, w.r, w.d_v, w.seq, w.decode_steps
    q = inputs.normal_bf16((B, H, S, r), w.seed + 1, device=device)
    k = inputs.normal_bf16((B, H, S, r), w.seed + 2, device=device)
    v = inputs.normal_bf16((B, H, S, dv), w.seed + 3, device=device)
    pre = torch.empty(B, H, S, dv, dtype=torch.float32, device=device)
    cache = tb.ThinKeyCache.allocate(B, H, H, r, dv, capacity=S + T, device=device)
    qd = inputs.normal_bf16((T, B, H, r), w.seed + 4, device=device)
    kd = inputs.normal_bf16((T, B, H, 1, r), w.seed + 5, device=device)
    vd = inputs.normal_bf16((T, B, H, 1, dv), w.seed + 6, device=device)
    out = torch.empty(T, B, H, dv, dtype=torch.float32, device=device)
    ws = tb.decode_workspace(cache.desc, S + T, device=device)
    zero = torch.zeros(B, dtype=torch.int32, device=device)
    lens = [torch.full((B,), S + t, dtype=torch.int32, device=device) for t in range(T + 1)]

    kd1 = kd.view(T, B, H, r)
    vd1 = vd.view(T, B, H, dv)

    def layer(_):
        tb.tk_attn_prefill(q, k, v, pre)
        tb.tk_kv_append(cache, k, v, zero)
        for t in range(T):
            tb.tk_attn_decode_append(cache, qd[t], kd1[t], vd1[t], lens[t], S + T, out[t], ws)

    sec = graph_time(torch, layer, iters, 3, max_graph=4) / iters
    flops = cm.prefill_flops(B, H, S, r, dv)
    kv = sum(cm.decode_kv_bytes([S + t + 1] * B, H, r, dv) for t in range(T))
    return {"layer_us": sec * 1e6, "launches_per_layer": 2 + T,
            "decode_tokens_per_s": B * T / sec, "prefill_flops": flops, "decode_kv_bytes": kv}


# ----------------------------------------------------------------------------- CPU oracle legs

CPU_CHILD = r"""
import json, sys, time, os
sys.path.insert(0, os.environ["TK_ROOT"])
import torch
from oracle import attention as oa
from oracle import cache as oc
from oracle.attention import bf16_bits_to_f64
from paper_2603_04427_gb300 import inputs, cost_model as cm
spec = json.loads(sys.argv[1])
f = lambda t: bf16_bits_to_f64(t.view(torch.int16).numpy())
seed, reps, warm, r, dv = spec["seed"], spec["reps"], spec["warm"], spec["r"], spec["dv"]
scale = 1.0 / r ** 0.5
if spec["mode"] == "decode":
    # a bounded sample: n_groups (sequence, kv head) groups of the workload, G query heads each
    n, L, G, kf = spec["groups"], spec["L"], spec["G"], spec.get("k", "bf16")
    kb = inputs.normal_bf16((1, n, L, r), seed + 1)
    v = f(inputs.normal_bf16((1, n, L, dv), seed + 2))
    q = f(inputs.normal_bf16((1, n * G, r), seed + 3))
    if kf == "bf16":
        k, sc, kbytes, sbytes = f(kb), None, 2, 0
    else:   # the oracle's own quantiser, before timing
        quant = oc.quantize_int8_per_token if kf == "int8" else oc.quantize_int4_per_token
        k, sc = quant(kb.float().numpy())
        kbytes, sbytes = (1, 4) if kf == "int8" else (0.5, 4)
    work = lambda: oa.attention_decode(q, k, v, [L], scale, k_scale=sc)
    amount = cm.decode_kv_bytes([L] * n, 1, r, dv, k_bytes=kbytes, k_scale_bytes=sbytes)
elif spec["mode"] == "decode_seq":
    # groups of different context lengths, built and timed one after the other
    G, kf, el, amount = spec["G"], spec.get("k", "bf16"), 0.0, 0
    print("ready", flush=True)
    sys.stdin.readline()
    for i, L in enumerate(spec["Ls"]):
        kb = inputs.normal_bf16((1, 1, L, r), seed + 10 * i + 1)
        v = f(inputs.normal_bf16((1, 1, L, dv), seed + 10 * i + 2))
        q = f(inputs.normal_bf16((1, G, r), seed + 10 * i + 3))
        if kf == "bf16":
            k, sc, kbytes, sbytes = f(kb), None, 2, 0
        else:
            quant = oc.quantize_int8_per_token if kf == "int8" else oc.quantize_int4_per_token
            k, sc = quant(kb.float().numpy())
            kbytes, sbytes = (1, 4) if kf == "int8" else (0.5, 4)
        t0 = time.perf_counter()
        oa.attention_decode(q, k, v, [L], scale, k_scale=sc)
        el += time.perf_counter() - t0
        amount += cm.decode_kv_bytes([L], 1, r, dv, k_bytes=kbytes, k_scale_bytes=sbytes)
    print(json.dumps({"sec": el, "reps": 1, "amount": amount}))
    sys.exit(0)
else:
    # a bounded sample of prefill: query rows row0 .. row0 + n - 1 of one causal head
    row0, n = spec["row0"], spec["rows"]
    q = f(inputs.normal_bf16((n, r), seed + 1))
    k = f(inputs.normal_bf16((row0 + n, r), seed + 2))
    v = f(inputs.normal_bf16((row0 + n, dv), seed + 3))
    work = lambda: oa.attention_head(q, k, v, scale, causal_offset=row0)
    amount = sum(i + 1 for i in range(row0, row0 + n)) * 2 * (r + dv)
print("ready", flush=True)   # inputs built; the timed work starts on the parent's word
sys.stdin.readline()
for _ in range(warm):
    work()
t0 = time.perf_counter()
for _ in range(reps):
    work()
el = time.perf_counter() - t0
print(json.dumps({"sec": el, "reps": reps, "amount": amount * reps}))
"""


def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def _run_cpu_children(specs):
    """Fresh single-threaded oracle processes, one per spec, built first and then
    started together; returns their results (seconds, repetitions, amount of work)."""
    env = dict(os.environ, TK_ROOT=ROOT, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1",
               MKL_NUM_THREADS="1", CUDA_VISIBLE_DEVICES="")
    children = [subprocess.Popen([sys.executable, "-c", CPU_CHILD, json.dumps(sp)], env=env,
                                 text=True, stdin=subprocess.PIPE, stdout=subprocess.PIPE,
                                 stderr=subprocess.PIPE) for sp in specs]
    try:
        for c in children:   # every child has built its inputs
            if c.stdout.readline().strip() != "ready":
                raise RuntimeError(c.stderr.read()[-2000:])
        for c in children:
            c.stdin.write("go\n")
            c.stdin.flush()
        outs = [c.communicate(timeout=900) for c in children]
    finally:
        for c in children:
            if c.poll() is None:
                c.kill()
    for c, (o, e) in zip(children, outs):
        if c.returncode != 0:
            raise RuntimeError(e[-2000:])
    return [json.loads(o.strip().splitlines()[-1]) for o, _ in outs]


def cpu_oracle_decode(w, n_groups: int, reps: int, warmup: int = 1, procs: int = 1, L=None,
                      k_fmt=None, r=None):
    """Time `reps` oracle decodes of a sample of the workload: `procs` fresh
    single-threaded processes, each on its share of the n_groups (sequence, kv
    head) groups, start their timed loops together; throughput = all their
    bytes / the slowest one's time."""
    procs = max(1, min(procs, n_groups))
    shares = [n_groups // procs + (1 if k < n_groups % procs else 0) for k in range(procs)]
    L = L or w.seq
    r = r or w.r
    k_fmt = k_fmt or ("int8" if w.k_int8 else "bf16")
    ds = _run_cpu_children([dict(mode="decode", seed=w.seed + 7 * k, reps=reps, warm=warmup, r=r,
                                 dv=w.d_v, groups=share, L=L, G=w.h_q // w.h_kv, k=k_fmt)
                            for k, share in enumerate(shares)])
    sec = max(d["sec"] for d in ds)
    return {"value": sum(d["amount"] for d in ds) / sec / 1e9, "unit": "GB/s", "cores": procs,
            "kind": "oracle", "sec": sec, "reps": reps,
            "sample": f"{n_groups} of {w.batch * w.h_kv} (sequence, kv-head) groups x "
                      f"{w.h_q // w.h_kv} query heads at context {L} ({k_fmt} keys, r={r}), "
                      f"{reps} timed repetitions ({sec:.1f} s) by {procs} concurrent "
                      f"single-threaded processes; fp64 numpy, inputs converted before timing"}


def cpu_oracle_prefill(w, rows: int, reps: int, procs: int, warmup: int = 1):
    """Time the oracle's causal prefill on a sample of the workload: process p computes
    `rows` consecutive query rows of one head, its blocks spread evenly over the
    sequence (so the sample holds short and long rows); throughput = the unmasked
    pairs' FLOPs (2 (r + d_v) per pair) of all processes / the slowest one's time."""
    S = w.seq
    starts = [((S - rows) * p // max(1, procs - 1)) // 16 * 16 for p in range(procs)]
    ds = _run_cpu_children([dict(mode="prefill", seed=w.seed + 7 * p, reps=reps, warm=warmup,
                                 r=w.r, dv=w.d_v, row0=r0, rows=rows)
                            for p, r0 in enumerate(starts)])
    sec = max(d["sec"] for d in ds)
    flops = sum(d["amount"] for d in ds)
    total = w.batch * w.h_q * S * (S + 1) // 2 * 2 * (w.r + w.d_v)
    return {"value": flops / sec / 1e12, "unit": "TFLOP/s", "cores": procs, "kind": "oracle",
            "sec": sec, "reps": reps,
            "full_workload_s_extrapolated": total / (flops / sec) if flops else None,
            "sample": f"{procs} blocks of {rows} consecutive causal query rows (one head each, "
                      f"starting rows spread over 0..{S - rows}) of the {w.batch}x{w.h_q}-head "
                      f"S={S} prefill, {reps} timed repetitions ({sec:.1f} s) by {procs} "
                      f"concurrent single-threaded processes; fp64 numpy"}


def cpu_oracle_workloads():
    """The oracle's time on every workload (fp64 numpy, all host cores): measured in
    full where that takes seconds, else on a stated sample and extrapolated by the
    workload's work.  Reported in one JSON line by ``bench.py --only cpu``."""
    from paper_2603_04427_gb300 import inputs
    from paper_2603_04427_gb300 import workloads as wl
    cores = host_cores()
    res = {}

    def spread(items, procs):
        return [items[p::procs] for p in range(procs) if items[p::procs]]

    # GPT-2-small layer: 12 heads' causal prefill of 256 rows, then 32 decode steps
    g = wl.GPT2_LAYER
    pre = _run_cpu_children([dict(mode="prefill", seed=g.seed + p, reps=1, warm=1, r=g.r, dv=g.d_v,
                                  row0=0, rows=g.seq) for p in range(g.h_q)])
    steps = [g.seq + t + 1 for t in range(g.decode_steps)]
    dec = _run_cpu_children([dict(mode="decode_seq", seed=g.seed + 50 + p, reps=1, warm=0, r=g.r,
                                  dv=g.d_v, G=1, Ls=steps) for p in range(g.h_q)])
    res[g.name] = {"sec": max(d["sec"] for d in pre) + max(d["sec"] for d in dec),
                   "cores": g.h_q, "how": "measured in full (one process per head)"}
    # Mistral GQA decode: all 128 (sequence, kv head) groups
    m = wl.MISTRAL_GQA_DECODE
    d = cpu_oracle_decode(m, m.batch * m.h_kv, 1, 1, min(cores, m.batch * m.h_kv))
    res[m.name] = {"sec": d["sec"], "cores": d["cores"], "how": "measured in full"}
    # 7B prefill: blocks of 512 query rows spread over the sequence, extrapolated by FLOPs
    p7 = cpu_oracle_prefill(wl.MHA7B_PREFILL, 512, 1, cores)
    res[wl.MHA7B_PREFILL.name] = {"sec": p7["full_workload_s_extrapolated"], "cores": cores,
                                  "how": "extrapolated from " + p7["sample"]}
    # paged long-context decode: all 32 (sequence, kv head) groups at their drawn lengths
    pw = wl.PAGED_LONG_DECODE
    lens = inputs.uniform_lengths(pw.batch, pw.seq_range[0], pw.seq_range[1], seed=pw.seed)
    items = [lens[b] for b in range(pw.batch) for _ in range(pw.h_kv)]
    dd = _run_cpu_children([dict(mode="decode_seq", seed=pw.seed + 13 * p, reps=1, warm=0, r=pw.r,
                                 dv=pw.d_v, G=pw.h_q // pw.h_kv, Ls=part)
                            for p, part in enumerate(spread(items, min(cores, len(items))))])
    res[pw.name] = {"sec": max(x["sec"] for x in dd), "cores": len(dd),
                    "how": "measured in full (gathered contexts; the oracle's gather not timed)"}
    # int8 keys, B=64, context 32768: two groups per core, extrapolated to all 512 groups
    iw = wl.INT8_DECODE
    n_s = 2 * cores
    dd = _run_cpu_children([dict(mode="decode_seq", seed=iw.seed + 13 * p, reps=1, warm=0, r=iw.r,
                                 dv=iw.d_v, G=iw.h_q // iw.h_kv, k="int8", Ls=[iw.seq, iw.seq])
                            for p in range(cores)])
    sec = max(x["sec"] for x in dd)
    res[iw.name] = {"sec": sec * iw.batch * iw.h_kv / n_s, "cores": cores,
                    "how": f"extrapolated from {n_s} of {iw.batch * iw.h_kv} (sequence, kv head) "
                           f"groups ({sec:.2f} s, two per core)"}
    return res


def run_reference(args, rank):
    """--impl reference: the fp64 CPU oracle on the headline workload, W + K steps.

    Each step is the oracle's decode over a sample of the workload's
    (sequence, kv head) groups, sized from a short calibration so that the
    whole run stays within about two minutes.
    """
    from paper_2603_04427_gb300 import workloads as wl
    w = wl.MISTRAL_GQA_DECODE
    if rank != 0:
        return
    cal = cpu_oracle_decode(w, 1, 5)
    t_group = cal["sec"] / cal["reps"]
    procs = min(host_cores(), w.batch * w.h_kv)
    n_groups = int(max(1, min(w.batch * w.h_kv, procs * 120.0 / (args.steps + args.warmup) / t_group)))
    res = cpu_oracle_decode(w, n_groups, args.steps, args.warmup, procs)
    line = {"impl": "reference", "metric": METRIC, "value": res["value"], "unit": "GB/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": res["sec"] / args.steps * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": dict(w.as_config(), sample_groups=n_groups),
            "cpu_baseline": res,
            "e2e": {"value": res["value"], "unit": "GB/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def max_over_ranks(dist, values, device):
    """Element-wise maximum of `values` over all ranks (the slowest rank's times);
    `values` unchanged on a single process (dist None)."""
    if dist is None:
        return [float(x) for x in values]
    import torch
    t = torch.tensor([float(x) for x in values], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(x) for x in t]


# ----------------------------------------------------------------------------- main

def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20000)
    ap.add_argument("--warmup", type=int, default=200)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--headline-only", action="store_true",
                    help="skip the secondary workloads and the CPU baseline")
    ap.add_argument("--only", choices=("decode", "prefill", "chunked", "chunked-r", "backward", "gpt2",
                                       "paged", "int8", "cpu"),
                    help="run one secondary workload alone (for profiling) and print its result; "
                         "cpu: the oracle's time on every workload")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, rank)
        return
    if args.only == "cpu":
        print(json.dumps({"only": "cpu", "oracle_seconds": cpu_oracle_workloads()}), flush=True)
        return

    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2603_04427_gb300 import binding as tb
    from paper_2603_04427_gb300 import cost_model as cm
    from paper_2603_04427_gb300 import workloads as wl

    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=device)
    peaks, peak_src = load_peaks()
    w = wl.MISTRAL_GQA_DECODE
    if args.only:
        res = {"only": args.only}
        if args.only == "prefill":
            res.update(measure_prefill(wl.MHA7B_PREFILL, args.steps, device, torch))
        elif args.only == "backward":
            res.update(measure_backward(wl.MHA7B_PREFILL, args.steps, device, torch))
        elif args.only == "chunked":
            for kf in ("bf16", "int8", "int4"):
                res[kf] = measure_chunked_prefill(wl.CHUNKED_PREFILL, args.steps, device, torch, k_fmt=kf)
        elif args.only == "chunked-r":
            # the same chunk at every thin-key width, bf16 and int8 keys
            import dataclasses
            rows = []
            for r in (16, 32, 64, 128):
                cw = dataclasses.replace(wl.CHUNKED_PREFILL, r=r)
                for kf in ("bf16", "int8"):
                    cp = measure_chunked_prefill(cw, args.steps, device, torch, k_fmt=kf)
                    rows.append([r, kf, round(cp["ms"], 4), round(cp["tflops"], 1),
                                 round(cp["tflops"] / peaks["bf16_tflops"], 4)])
            res["sweep"] = {"cols": ["r", "k_dtype", "ms", "TFLOP/s", "frac"], "rows": rows}
        elif args.only == "gpt2":
            res.update(measure_gpt2_layer(wl.GPT2_LAYER, args.steps, device, torch))
        elif args.only == "decode":
            # the headline workload's decode kernel alone (tk_attn_decode), for profiling
            drig = DecodeRig(w, device)
            sd = measure_decode(drig, args.steps, args.warmup, mode="decode")
            res.update(decode_kernel_us=sd * 1e6, kv_bytes=drig.kv_bytes,
                       frac=(drig.kv_bytes + drig.io_bytes) / sd / 1e9 / peaks["hbm_gbs"])
        else:
            ow = wl.PAGED_LONG_DECODE if args.only == "paged" else wl.INT8_DECODE
            orig = DecodeRig(ow, device, copies=1)
            sd = measure_decode(orig, args.steps, args.warmup, mode="decode")
            res.update(decode_kernel_us=sd * 1e6, kv_bytes=orig.kv_bytes,
                       frac=(orig.kv_bytes + orig.io_bytes) / sd / 1e9 / peaks["hbm_gbs"])
        print(json.dumps(res), flush=True)
        return

    rig = DecodeRig(w, device)
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    clocks = ClockSampler(local)
    clocks.start()
    timing = {}
    # the headline: K-step blocks replayed for at least a second, median block
    sec_step = measure_decode(rig, args.steps, args.warmup, mode="fused", min_seconds=1.0,
                              info=timing)
    sec_two = measure_decode(rig, args.steps, args.warmup, mode="append", min_seconds=0.2)
    sec_dec = measure_decode(rig, args.steps, args.warmup, mode="decode", min_seconds=0.3)
    torch.cuda.synchronize()
    clk = clocks.stop()
    sec_step, sec_dec, sec_two = max_over_ranks(dist, (sec_step, sec_dec, sec_two), device)
    n = world
    value = n * rig.kv_bytes / sec_step / 1e9
    e2e_dt, h2d, d2h = measure_decode_e2e(rig, min(args.steps, 5000))
    e2e_eager_dt, _, _ = measure_decode_e2e(rig, min(args.steps, 2000), graph=False)
    e2e_dt, e2e_eager_dt = max_over_ranks(dist, (e2e_dt, e2e_eager_dt), device)
    achieved = (rig.kv_bytes + rig.io_bytes) / sec_dec / 1e9
    dec_hash = source_hash("decode.cu", "common.cuh", "kv_row.cuh", "kernels.h", "widen.cuh")
    line = {
        "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": n, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": sec_step * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": dict(w.as_config(), storage="bf16 K/V, fp32 accumulate, fp32 out",
                       step="tk_attn_decode_append: the new token of every sequence is "
                            "appended inside the decode launch",
                       l2=f"rotating {len(rig.copies)} cache copies "
                          f"({len(rig.copies) * rig.kv_bytes / 1e6:.0f} MB > 4x L2)",
                       parallelism=f"replicas x{n}" if n > 1 else "single GPU"),
        "tokens_per_s": n * w.batch / sec_step,
        "two_call_step_us": sec_two * 1e6,
        "kv_bytes_per_step": rig.kv_bytes,
        "hbm_frac_of_measured_peak": value / peaks["hbm_gbs"],
        "roofline": {"kernel": "decode_kernel<32,128,4,bf16>", "bound": "hbm",
                     "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                     "frac": achieved / peaks["hbm_gbs"], "peak_source": peak_src,
                     "launch_us": sec_dec * 1e6,
                     "bytes_per_launch": rig.kv_bytes + rig.io_bytes,
                     "traffic": recorded_traffic("decode", w.name, dec_hash)},
        "e2e": {"value": n * rig.kv_bytes / e2e_dt / 1e9, "unit": "GB/s",
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "ms_per_step": e2e_dt * 1e3,
                "ms_per_step_without_graph": e2e_eager_dt * 1e3,
                "how": "per step: the step's q, k_new, v_new from one page-locked host "
                       "buffer (tk_copy_async) and the fused append + decode, prepared once "
                       "by the binding and recorded as one CUDA graph (tk_graph_begin / "
                       "tk_graph_end), replayed by one tk_graph_launch per step; the kernel "
                       "writes the output into page-locked host memory (zero-copy); host "
                       "synchronisation every step"},
        "gpu_launches": args.steps * timing.get("blocks", 1),
        "timing": {"blocks": timing.get("blocks"), "timed_region_s": timing.get("timed_region_s"),
                   "launches_per_step": 1,
                   "ms_per_step": f"median over blocks of {args.steps} steps (CUDA events)"},
        "clocks": clk,
    }
    del rig
    torch.cuda.empty_cache()

    if rank == 0 and not args.headline_only:
        def r3(x):
            return float(f"{x:.4g}")
        if n == 1:
            try:
                cal = cpu_oracle_decode(w, 1, 5)
                procs = min(host_cores(), w.batch * w.h_kv)
                groups = min(w.batch * w.h_kv, 16 * procs)
                reps = max(1, int(10.0 / (cal["sec"] / cal["reps"] * groups / procs)))
                line["cpu_baseline"] = cpu_oracle_decode(w, groups, reps, procs=procs)
            except Exception as e:  # reported, not fatal
                line["cpu_baseline"] = {"error": str(e)[-300:]}
        else:
            line["cpu_baseline"] = None
        extra = {}
        gw = wl.GPT2_LAYER
        extra[gw.name] = dict(gw.as_config(), **measure_gpt2_layer(gw, 50, device, torch))
        # paged long-context decode
        pl = wl.PAGED_LONG_DECODE
        prig = DecodeRig(pl, device, copies=1)
        s = measure_decode(prig, 200, 20, mode="fused")
        sd = measure_decode(prig, 200, 20, mode="decode")
        extra[pl.name] = dict(pl.as_config(), seq_lens=prig.lens, kv_bytes=prig.kv_bytes,
                              step_us=r3(s * 1e6), gbs=r3(prig.kv_bytes / s / 1e9),
                              decode_kernel_us=r3(sd * 1e6),
                              decode_kernel_frac=r3((prig.kv_bytes + prig.io_bytes) / sd / 1e9 / peaks["hbm_gbs"]))
        del prig
        torch.cuda.empty_cache()
        # quantised keys, B=64, context 32768, and the r sweep (int4, int8 and bf16 keys)
        iw = wl.INT8_DECODE
        rows = []
        for r in iw.r_sweep:
            for kf in ("int4", "int8", "bf16"):
                if kf == "int4" and r < 32:
                    continue
                rr = DecodeRig(iw, device, copies=1, k_fmt=kf, r=r)
                s = measure_decode(rr, 50, 5, mode="fused")
                sd = measure_decode(rr, 50, 5, mode="decode")
                rows.append([r, kf, rr.kv_bytes, r3(s * 1e6), r3(rr.kv_bytes / s / 1e9), r3(sd * 1e6),
                             r3((rr.kv_bytes + rr.io_bytes) / sd / 1e9 / peaks["hbm_gbs"])])
                del rr
                torch.cuda.empty_cache()
        extra[iw.name] = dict(iw.as_config(), sweep={
            "cols": ["r", "k_dtype", "kv_bytes", "step_us", "GB/s", "decode_kernel_us",
                     "decode_kernel_frac"], "rows": rows})
        # training backward and chunked prefill of the 7B shape
        pw = wl.MHA7B_PREFILL
        bw = measure_backward(pw, 10, device, torch)
        bname = pw.name.replace("prefill", "backward")
        extra[bname] = dict(
            pw.as_config(), workload=bname, kernel="bwd_tc_kernel<32,128> (tcgen05)", ms=r3(bw["ms"]),
            tflops=r3(bw["tflops"]), frac=r3(bw["tflops"] / peaks["bf16_tflops"]),
            flops_per_call=bw["flops_per_call"], launches=bw["launches"])
        cw = wl.CHUNKED_PREFILL
        for kf in ("bf16", "int8"):
            cp = measure_chunked_prefill(cw, 20, device, torch, k_fmt=kf)
            name = cw.name if kf == "bf16" else cw.name + "_int8_keys"
            extra[name] = dict(cw.as_config(), workload=name, k_dtype=kf, ms=r3(cp["ms"]),
                               tflops=r3(cp["tflops"]),
                               frac=r3(cp["tflops"] / peaks["bf16_tflops"]),
                               append_ms=r3(cp["append_ms"]), flops_per_call=cp["flops_per_call"],
                               launches=cp["launches"])
        line["workloads"] = extra
        # the causal prefill half of the metric, last on the line
        pf = measure_prefill(pw, 20, device, torch)
        pre = dict(pw.as_config(), kernel="prefill_kernel<32,128> (tcgen05)")
        if "tflops" in pf:
            pre.update(ms=r3(pf["ms"]), tflops=r3(pf["tflops"]), flops_per_launch=pf["flops_per_launch"],
                       roofline={"bound": "tensor", "achieved": r3(pf["tflops"]),
                                 "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
                                 "frac": r3(pf["tflops"] / peaks["bf16_tflops"]),
                                 "peak_source": peak_src,
                                 "traffic": recorded_traffic("prefill", pw.name, source_hash(
                                     "prefill.cu", "common.cuh", "tc05.cuh", "widen.cuh",
                                     "kernels.h"))})
        else:
            pre.update(pf)
        if n == 1:
            try:
                procs = host_cores()
                # calibrate on the same blocks (the last one, near row S, is the slowest)
                cal = cpu_oracle_prefill(pw, 512, 1, procs, warmup=0)
                reps = max(1, int(10.0 / cal["sec"]))
                cb = cpu_oracle_prefill(pw, 512, reps, procs)
                pre["cpu_baseline"] = {k: (r3(v) if isinstance(v, float) else v) for k, v in cb.items()}
            except Exception as e:  # reported, not fatal
                pre["cpu_baseline"] = {"error": str(e)[-300:]}
        line["prefill"] = pre
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist:
        dist.barrier()
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
