"""Benchmark: batch-1 decode of the Llama-2-7B-shaped stack, every tensor-parallel shard on one GPU.

One step = one decode token through all 32 layers: for each layer every ATTN shard (4 of them),
the on-device combine, every FFN shard, the combine; then the KV lengths advance.  The token step
is one CUDA graph of vt_decode_token (one fused cooperative kernel, in which the shards of a block
run side by side, each with its own fp32 partial, and the combines add them in shard order)
replayed K times; the KV length runs 1024 -> 1151 and rewinds to 1024 every 128 steps (the
128-step schedule of the workload).  The K-step timed region is repeated until it covers
--min-timed-s seconds, so the clock sampler sees enough samples; ms_per_step is the median.

Printed: one JSON line (rank 0).  `value` is device-timed tokens/s with inputs resident in HBM;
`e2e` is the same metric through the C ABI with host buffers (token id H2D, hidden state D2H,
synchronised every step); `roofline` is the token kernel's achieved HBM bandwidth (algorithmic
bytes of the step over its time); `sharded_token` times the same token as per-shard kernels;
`cpu_baseline` is the CPU oracle timed on a bounded sample (all host threads, and one thread in
`value_1thread`); `prefill` is the 512-token prompt of the 7B prefill workload through the same
stack (tok/s and tensor-core rate, with the oracle's prefill in `prefill.cpu_baseline`);
`other_workloads` are the 13B (uneven 3-way, KV 2048) and 8B GQA (4-way, KV 4096) decode shapes
timed the same way.
`--impl reference` times the CPU oracle alone.
"""
from __future__ import annotations

import argparse
import json
import os
import subprocess
import sys
import tempfile
import threading
import time
from pathlib import Path

ROOT = Path(__file__).resolve().parent
sys.path.insert(0, str(ROOT))

import numpy as np  # noqa: E402

import synthetic  # noqa: E402

METRIC = "batch-1 decode tok/s (7B fp16, all shards on 1 GPU); % of HBM roofline"
WORKLOAD = ("llama2-7b-shaped batch-1 decode: 32 layers, D 4096, 32 heads x 128 (MHA), "
            "FFN 11008 SwiGLU; even 4-way TP (8 heads, 2752 FFN columns per shard), all shards on "
            "1 GPU: the shards of a block run side by side inside one launch, each keeping its own "
            "fp32 partial, combined in shard order; KV 1024 -> 1151 (128-step schedule)")
FALLBACK_HBM_GBS = 6800.0

# DRAM bytes (read + write) of one launch of the decode-token kernel, from one ncu capture of
# that kernel (mean of 12 launches of the 7B decode; profiles/k_decode_token_7b.md), and a
# digest of the sources the captured kernel was built from.  The line reports the bytes only
# while the sources still hash to that digest: a changed kernel reports null until recaptured.
K_TOKEN_DRAM_BYTES_PER_LAUNCH = 13_504_038_379
K_TOKEN_SOURCES = ("token_kernel.cuh", "token.cu", "token_v1.cu", "token_v2.cu", "internal.h", "device.cuh")
K_TOKEN_SOURCES_SHA256 = "dfeb75c0fa54e6a3"


def token_traffic_if_current():
    import hashlib
    h = hashlib.sha256()
    for f in K_TOKEN_SOURCES:
        h.update((ROOT / "paper_2607_07046_gb300" / "csrc" / f).read_bytes())
    return K_TOKEN_DRAM_BYTES_PER_LAUNCH if h.hexdigest()[:16] == K_TOKEN_SOURCES_SHA256 else None


def all_ranks_max(torch, x: float, device: str) -> float:
    """The maximum of x over the ranks of the process group (x itself on one process): the
    timed region's repeat count and its step time are taken as the slowest rank's."""
    if not (torch.distributed.is_available() and torch.distributed.is_initialized()):
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def replicas_tok_s(world: int, ms_per_step: float) -> float:
    """Whole-job decode rate: every rank decodes its own token stream (a replica), so the job
    makes `world` tokens per step of the slowest rank."""
    return world * 1000.0 / ms_per_step


def measured_peaks():
    p = ROOT / "MEASURED_PEAKS.json"
    if p.exists():
        d = json.loads(p.read_text())
        return float(d["hbm_gbs"]), float(d.get("bf16_tflops", 1900.0)), \
            float(d.get("bf16_tflops_sustained", 1700.0)), "measured"
    return FALLBACK_HBM_GBS, 1900.0, 1700.0, "fallback"


# ------------------------------------------------------------------ clocks sampler

class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "25"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except FileNotFoundError:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.15)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        if not self.path or not os.path.exists(self.path):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no nvidia-smi"]}
        rows = []
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((float(parts[1]), float(parts[2]), float(parts[3]), parts[5:9]))
            except ValueError:
                continue
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        load = [r for r in rows if r[2] > 200.0] or rows
        sm = sorted(r[0] for r in load)
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in load for i, v in enumerate(r[3]) if v == "Active"})
        return {"sm_mhz": sm[len(sm) // 2], "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(load), "power_w_max": max(r[2] for r in rows)}


# ------------------------------------------------------------------ workload

def shapes_for(vt, wl, max_seq):
    return vt.make_shapes(wl.n_layers, wl.d_model, wl.n_heads, wl.n_kv_heads, wl.d_head, wl.d_ffn,
                          wl.vocab, max_seq, wl.rms_eps, wl.rope_theta)


def decode_bytes_per_token(wl, kv_mean):
    """Algorithmic HBM bytes of one decode token: every shard weight once, the cache read at the
    mean length (+1 for the new token), the new K/V row written."""
    D, H, Hk, dh, F, L = wl.d_model, wl.n_heads, wl.n_kv_heads, wl.d_head, wl.d_ffn, wl.n_layers
    w = 2 * (D * (H + 2 * Hk) * dh + D * H * dh + 3 * D * F + 2 * D)
    kv = 2 * 2 * Hk * dh * (kv_mean + 1)
    return L * (w + kv)


def quant_bytes_per_token(wl, bits, kv_mean):
    """Algorithmic HBM bytes of one decode token with every shard block-quantized at `bits`: the
    codes (one byte per weight at 8 bits, half a byte at 4; rows padded to whole blocks of 32) and
    one fp16 scale per block of every projection, the layer's two RMSNorm gains (one buffer each,
    as in decode_bytes_per_token), the cache at the mean length."""
    D, H, Hk, dh, F, L = wl.d_model, wl.n_heads, wl.n_kv_heads, wl.d_head, wl.d_ffn, wl.n_layers
    cb = 1.0 if bits == 8 else 0.5

    def mat(rows, k):
        nb = (k + 31) // 32
        return rows * (nb * 32 * cb + nb * 2)

    w = 2.0 * 2 * D
    for (h0, h1), (c0, c1) in zip(wl.head_ranges, wl.ffn_ranges):
        hq, c = h1 - h0, c1 - c0
        hk = hq * Hk // H
        if hq:
            w += mat((hq + 2 * hk) * dh, D) + mat(D, hq * dh)
        if c:
            w += mat(2 * c, D) + mat(D, c)
    kv = 2 * 2 * Hk * dh * (kv_mean + 1)
    return int(L * (w + kv))


def kernels_per_token(wl):
    """Kernels of one vt_decode_token: per layer, 3 per non-empty ATTN shard (QKV GEMV,
    attention, O GEMV), 1 per non-empty FFN shard (fused FFN), 2 combines; 1 KV advance."""
    n = 0
    for (h0, h1), (c0, c1) in zip(wl.head_ranges, wl.ffn_ranges):
        n += 3 if h1 > h0 else 0
        n += 1 if c1 > c0 else 0
    return wl.n_layers * (n + 2) + 1


def cpu_baseline_decode(wl, layers=4, budget_s=12.0, max_tokens=512, budget_1thread_s=4.0, max_tokens_1thread=32):
    """The oracle (as it stands) on `layers` layers, decoding teacher-forced tokens from KV 1024
    until about `budget_s` seconds have passed on all host threads, then about `budget_1thread_s`
    seconds on one thread (continuing the same caches); tok/s is extrapolated to the full stack by
    the layer ratio."""
    import oracle
    threads = oracle.num_threads()
    L0 = wl.kv_len
    ws = [wl.layer_weights(l) for l in range(layers)]
    caches = [wl.kv_fill(l, L0, L0 + max_tokens + max_tokens_1thread + 1) for l in range(layers)]
    tokens = 0

    def run(budget, limit):
        nonlocal tokens
        t0 = time.perf_counter()
        done = 0
        while done < limit and (done < 1 or time.perf_counter() - t0 < budget):
            x = wl.hidden(1, stream=500 + tokens)
            for l in range(layers):
                _, x, _, _ = oracle.tp_layer(wl, ws[l], x, L0 + tokens, *caches[l])
            tokens += 1
            done += 1
        return done, time.perf_counter() - t0

    n_all, dt = run(budget_s, max_tokens)
    oracle.set_threads(1)
    try:
        n_one, dt1 = run(budget_1thread_s, max_tokens_1thread)
    finally:
        oracle.set_threads(threads)
    scale = wl.n_layers / layers
    return {"value": round(n_all / (dt * scale), 4), "unit": "tok/s", "cores": threads,
            "kind": "oracle",
            "sample": f"{n_all} teacher-forced decode tokens through layers 0-{layers - 1} of "
                      f"{wl.n_layers} from KV {L0}, 4-way TP shards, fp64 oracle; tok/s "
                      f"extrapolated x{scale:g} by layers",
            "seconds": round(dt, 2),
            "value_1thread": round(n_one / (dt1 * scale), 4),
            "sample_1thread": f"{n_one} further tokens on 1 thread (same layers and extrapolation)",
            "seconds_1thread": round(dt1, 2)}


def cpu_baseline_prefill(wl, layers=1):
    """The oracle (as it stands) on the whole prompt of the prefill workload through `layers`
    layers on all host threads; tok/s is extrapolated to the full stack by the layer ratio."""
    import oracle
    n = wl.prompt_len
    x = wl.hidden(n, stream=600)
    t0 = time.perf_counter()
    for l in range(layers):
        kc, vc = oracle.new_cache(wl, n)
        _, x, _, _ = oracle.tp_layer(wl, wl.layer_weights(l), x, 0, kc, vc)
    dt = time.perf_counter() - t0
    scale = wl.n_layers / layers
    return {"value": round(n / (dt * scale), 2), "unit": "tok/s", "cores": oracle.num_threads(),
            "kind": "oracle",
            "sample": f"the {n}-token prompt through layer(s) 0-{layers - 1} of {wl.n_layers}, 4-way TP "
                      f"shards, fp64 oracle; tok/s extrapolated x{scale:g} by layers",
            "seconds": round(dt, 2)}


def prefill_gemm_flops(wl, n):
    """Tensor-core FLOPs of an n-row prefill through the stack: QKV, O, gate/up and down
    projections of every shard (2 flops per multiply-add)."""
    D, H, Hk, dh, F = wl.d_model, wl.n_heads, wl.n_kv_heads, wl.d_head, wl.d_ffn
    return 2 * n * wl.n_layers * (D * (H + 2 * Hk) * dh + D * H * dh + 3 * D * F)


def prefill_attn_flops(wl, n):
    """Causal attention of an n-row prompt from position 0: QK^T and PV over i + 1 positions."""
    return 4 * wl.d_head * wl.n_heads * wl.n_layers * n * (n + 1) // 2


def run_prefill(vt, st, wl, stream, steps, warmup):
    """The 512-token prompt of the 7B prefill workload through every layer (vt_prefill_tokens: the
    shards of a block together, one launch per projection and one for the attention), captured
    with the embedding and a KV rewind as one CUDA graph."""
    import torch
    wp = synthetic.WORKLOADS[4]
    n, D = wp.prompt_len, wl.d_model
    ids = torch.from_numpy(wp.token_ids(n, stream=3)).cuda()
    x = torch.empty((n, D), dtype=torch.float16, device="cuda")
    y = torch.empty((n, D), dtype=torch.float16, device="cuda")
    vt.vt_kv_set_length(st.kv, -1, 0, stream)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(stream):
        with torch.cuda.graph(g, stream=stream):
            vt.vt_embed(st.model, ids, x, stream)
            vt.vt_prefill_tokens(st.part, st.kv, x, n, y, stream)
            vt.vt_kv_advance(st.kv, -1, -n, stream)
        for _ in range(warmup):
            g.replay()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(steps):
            g.replay()
        e1.record(stream)
    e1.synchronize()
    ms = e0.elapsed_time(e1) / steps
    finite = bool(torch.isfinite(y.float()).all().item())
    _, _, tf_sustained, peak_kind = measured_peaks()
    gemm = prefill_gemm_flops(wl, n)
    tflops = gemm / (ms * 1e-3) / 1e12
    n_dev = len(wl.head_ranges)
    # kernels per prompt: embedding, the first RMSNorm, per layer (QKV, O, gate/up and down GEMMs,
    # one launch each per 8 shards; the attention, one launch per 6 shards; two combines +
    # RMSNorm), KV advance and rewind
    launches = 2 + wl.n_layers * (4 * -(-n_dev // 8) + -(-n_dev // 6) + 2) + 2
    return {
        "workload": f"llama2-7b-shaped prefill: {n}-token prompt (seeded ids, embedding gather), "
                    f"{wl.n_layers} layers, even {n_dev}-way TP on 1 GPU (one grouped GEMM launch per "
                    f"projection covers every shard, each with its own fp32 partial)",
        "value": round(n / (ms * 1e-3), 1), "unit": "tok/s", "ms_per_prompt": round(ms, 4),
        "steps": steps, "warmup": warmup,
        "gemm_tflop_per_prompt": round(gemm / 1e12, 4),
        "attn_gflop_per_prompt": round(prefill_attn_flops(wl, n) / 1e9, 2),
        "roofline": {"bound": "tensor", "achieved": round(tflops, 1), "peak": tf_sustained,
                     "unit": "TFLOP/s", "frac": round(tflops / tf_sustained, 4),
                     "peak_kind": f"{peak_kind} sustained bf16 dense (fp16 dense has the same nominal rate)",
                     "note": "GEMM FLOPs over the whole prompt time (RMSNorm, attention, combines "
                             "included): a lower bound on the GEMM kernels' own rate"},
        "gpu_launches": launches * steps, "finite": finite,
    }


class TokenSchedule:
    """Replays one decode token per step as a CUDA graph of `entry` (a whole-token entry point):
    g_tok is one token; g_rew is one token followed by a rewind of every KV length by the
    schedule length (the last step of each 128-step schedule 1024 -> 1151)."""

    def __init__(self, vt, st, entry, xin, xout, stream, sched, kv_len):
        import torch
        self.vt, self.st, self.stream, self.sched, self.kv_len = vt, st, stream, sched, kv_len
        self.g_tok, self.g_rew = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
        with torch.cuda.stream(stream):
            with torch.cuda.graph(self.g_tok, stream=stream):
                entry(st.part, st.kv, xin, xout, stream)
            with torch.cuda.graph(self.g_rew, stream=stream):
                entry(st.part, st.kv, xin, xout, stream)
                vt.vt_kv_advance(st.kv, -1, -sched, stream)
        self.reset()

    def reset(self):
        # replays advance the device lengths (captures leave them and the host mirror alone):
        # put both back at kv_len
        self.vt.vt_kv_set_length(self.st.kv, -1, self.kv_len, self.stream)
        self.pos = 0

    def step(self):
        self.pos += 1
        if self.pos == self.sched:
            self.g_rew.replay()
            self.pos = 0
        else:
            self.g_tok.replay()


def time_tokens(torch, sch, stream, steps, warmup):
    with torch.cuda.stream(stream):
        for _ in range(warmup):
            sch.step()
    stream.synchronize()
    sch.reset()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e0.record(stream)
        for _ in range(steps):
            sch.step()
        e1.record(stream)
    e1.synchronize()
    return e0.elapsed_time(e1) / steps


def run_decode(args, rank, world):
    import torch

    from paper_2607_07046_gb300 import build as vt_build
    from paper_2607_07046_gb300 import vt
    from paper_2607_07046_gb300.stack import Stack

    vt_build.build()
    wl = synthetic.WORKLOADS[2]
    if args.layers:
        import dataclasses
        wl = dataclasses.replace(wl, n_layers=args.layers)
    torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", 0)))
    sched = wl.decode_steps  # 128-step KV schedule 1024 -> 1151
    cap = wl.kv_len + sched + 8
    shapes = shapes_for(vt, wl, cap)
    stream = torch.cuda.Stream()
    t_setup = time.perf_counter()
    with torch.cuda.stream(stream):
        st = Stack(shapes, wl.layer_weights, wl.head_ranges, wl.ffn_ranges, cap,
                   embed=wl.embedding(), stream=stream)
    try:
        for l in range(wl.n_layers):
            kc, vc = wl.kv_fill(l, wl.kv_len)
            for d, (h0, h1) in enumerate(wl.head_ranges):
                vt.vt_kv_write_raw(st.kv, l, d, kc[h0:h1], vc[h0:h1])
        vt.vt_kv_set_length(st.kv, -1, wl.kv_len, stream)
        setup_s = time.perf_counter() - t_setup
        D = wl.d_model
        fused, why = vt.vt_decode_token_fused_available(st.part)
        ids = torch.from_numpy(wl.token_ids(1, stream=1)).cuda()
        xin = torch.empty(D, dtype=torch.float16, device="cuda")
        xout = torch.empty(D, dtype=torch.float16, device="cuda")
        with torch.cuda.stream(stream):
            vt.vt_embed(st.model, ids, xin, stream)
        stream.synchronize()
        sch = TokenSchedule(vt, st, vt.vt_decode_token, xin, xout, stream, sched, wl.kv_len)

        # warm-up steps, timed once to size the measurement: the timed region is exactly K steps,
        # repeated R times (R from the warm-up rate, the same on every rank) so that the clock
        # sampler sees at least ~10 samples at 25 ms; ms_per_step is the median repeat
        w0, w1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            w0.record(stream)
            for _ in range(args.warmup):
                sch.step()
            w1.record(stream)
        w1.synchronize()
        est_ms = w0.elapsed_time(w1) / max(args.warmup, 1)
        repeats = int(min(64, max(1, np.ceil(args.min_timed_s * 1e3 / max(est_ms * args.steps, 1e-3)))))
        if world > 1:
            repeats = int(all_ranks_max(torch, repeats, "cuda"))
        sch.reset()
        rep_ms = []
        with ClockSampler(torch.cuda.current_device()) as clk:
            for _ in range(repeats):
                if world > 1:
                    torch.distributed.barrier()
                torch.cuda.synchronize()
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                with torch.cuda.stream(stream):
                    e0.record(stream)
                    for _ in range(args.steps):
                        sch.step()
                    e1.record(stream)
                e1.synchronize()
                torch.cuda.synchronize()
                rep_ms.append(e0.elapsed_time(e1))
        ms = float(np.median(rep_ms))
        if world > 1:
            ms = all_ranks_max(torch, ms, "cuda")
        ms_per_step = ms / args.steps
        kv_status = vt.vt_kv_status(st.kv, clear=True)
        part_status = vt.vt_partition_status(st.part, clear=True)

        # -------------------------------------------------------------- e2e through host buffers
        sch.reset()
        ids_host = torch.from_numpy(wl.token_ids(max(args.steps, 1), stream=2)).pin_memory()
        ids_dev = torch.empty(1, dtype=torch.int32, device="cuda")
        out_host = torch.empty(D, dtype=torch.float16).pin_memory()
        e2e_steps = max(1, min(args.steps, 256))

        def e2e_step(i):
            ids_dev.copy_(ids_host[i:i + 1], non_blocking=True)
            vt.vt_embed(st.model, ids_dev, xin, stream)
            sch.step()
            out_host.copy_(xout, non_blocking=True)
            stream.synchronize()

        with torch.cuda.stream(stream):
            for i in range(min(3, e2e_steps)):
                e2e_step(i)
        sch.reset()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        with torch.cuda.stream(stream):
            for i in range(e2e_steps):
                e2e_step(i)
        e2e_s = (time.perf_counter() - t0) / e2e_steps
        if world > 1:
            e2e_s = all_ranks_max(torch, e2e_s, "cuda")
        e2e_finite = bool(np.isfinite(out_host.numpy().astype(np.float32)).all())

        # -------------------------------------------------------------- per-shard kernels, for context
        sharded_ms = None
        if args.sharded_steps > 0:
            sch2 = TokenSchedule(vt, st, vt.vt_decode_token_sharded, xin, xout, stream, sched, wl.kv_len)
            sharded_ms = time_tokens(torch, sch2, stream, args.sharded_steps, 3)
            del sch2
        sch.reset()
        prefill = run_prefill(vt, st, wl, stream, args.prefill_steps, 3) if args.prefill_steps > 0 else None
    finally:
        torch.cuda.synchronize()
        st.close()

    hbm, _, _, peak_kind = measured_peaks()
    kv_mean = wl.kv_len + (min(args.steps, sched) - 1) / 2.0
    step_bytes = decode_bytes_per_token(wl, kv_mean)
    value = replicas_tok_s(world, ms_per_step)
    achieved = step_bytes / (ms_per_step * 1e-3) / 1e9
    launches_per_token = 1 if fused else kernels_per_token(wl)
    line = {
        "metric": METRIC,
        "value": round(value, 3),
        "unit": "tok/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(ms_per_step, 5),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "fp16",
        "data": "synthetic (seeded N(0,0.02) fp16 weights, seeded N(0,(0.02*sqrt(D))^2) KV cache)",
        "config": {
            "workload": WORKLOAD,
            "kv_len_start": wl.kv_len,
            "kv_schedule_steps": sched,
            "partition": "heads 8/8/8/8, ffn 2752 x 4",
            "token_kernel": "fused: one cooperative kernel per token" if fused
                            else f"per-shard kernels ({why})",
            "graph": "one CUDA graph per token (vt_decode_token)",
            "l2": "no flush: the 13 GB of weights streamed per step exceed the 129 MB L2",
            "parallelism": f"replicas x{world}" if world > 1 else "1 GPU",
            "hbm_bytes_per_step": int(step_bytes),
        },
        "roofline": {
            "bound": "hbm",
            "kernel": ("k_decode_token (the whole token: every shard of every layer in one "
                       "cooperative launch, so the kernel's launch time is the step time)") if fused
                      else "the whole token step (per-shard kernels)",
            "achieved": round(achieved, 1),
            "peak": hbm,
            "unit": "GB/s",
            "frac": round(achieved / hbm, 4),
            "peak_kind": f"{peak_kind} copy bandwidth",
            "bytes_per_launch": int(step_bytes) if fused else None,
            "launch_ms": round(ms_per_step, 5),
            "traffic": token_traffic_if_current() if fused and not args.layers else None,
        },
        "e2e": {"value": round(world / e2e_s, 3), "unit": "tok/s", "h2d_bytes_per_step": 4,
                "d2h_bytes_per_step": 2 * D, "finite": e2e_finite},
        "timed_repeats": repeats,
        "ms_per_step_repeats": [round(r / args.steps, 5) for r in rep_ms],
        "gpu_launches": launches_per_token * args.steps + (args.steps // sched),
        "device_status": {"kv": kv_status, "partition": part_status},
        "setup_s": round(setup_s, 1),
    }
    if sharded_ms is not None:
        # the same token through the per-shard entry points: the same bytes at its own schedule's
        # mean KV length
        sh_bytes = decode_bytes_per_token(wl, wl.kv_len + (min(args.sharded_steps, sched) - 1) / 2.0)
        sh_achieved = sh_bytes / (sharded_ms * 1e-3) / 1e9
        line["sharded_token"] = {"ms_per_step": round(sharded_ms, 5), "value": round(1000.0 / sharded_ms, 3),
                                 "unit": "tok/s", "steps": args.sharded_steps,
                                 "note": "vt_decode_token_sharded: per-shard kernels with PDL, for context",
                                 "roofline": {"bound": "hbm",
                                              "kernel": "the whole token step (k_gemv, k_attn_decode, k_ffn and "
                                                        "k_combine for every shard and block)",
                                              "achieved": round(sh_achieved, 1), "peak": hbm, "unit": "GB/s",
                                              "frac": round(sh_achieved / hbm, 4),
                                              "peak_kind": f"{peak_kind} copy bandwidth",
                                              "bytes_per_step": int(sh_bytes)}}
    if prefill is not None:
        line["prefill"] = prefill
        line["gpu_launches"] += prefill["gpu_launches"]
    return line, clk.summary()


def run_decode_workload(cid, steps, warmup, bits=16, layers=0):
    """Decode tok/s of one more workload (the 13B uneven 3-way and the 8B GQA 4-way shapes), timed
    like the headline one: vt_decode_token replayed as a CUDA graph over the workload's KV schedule
    (kv_len -> kv_len + decode_steps - 1, then rewound), inputs resident on the device.  layers > 0:
    only the first `layers` layers (a small case for profiling)."""
    import dataclasses

    import torch

    from paper_2607_07046_gb300 import vt
    from paper_2607_07046_gb300.stack import Stack

    wl = synthetic.WORKLOADS[cid]
    if layers:
        wl = dataclasses.replace(wl, n_layers=layers)
    sched = wl.decode_steps
    cap = wl.kv_len + sched + 8
    stream = torch.cuda.Stream()
    t_setup = time.perf_counter()
    prec = None if bits == 16 else (lambda l, d, b: bits)
    with torch.cuda.stream(stream):
        st = Stack(shapes_for(vt, wl, cap), wl.layer_weights, wl.head_ranges, wl.ffn_ranges, cap, stream=stream,
                   precision=prec)
    try:
        g = wl.n_heads // wl.n_kv_heads
        for l in range(wl.n_layers):
            kc, vc = wl.kv_fill(l, wl.kv_len)
            for d, (h0, h1) in enumerate(wl.head_ranges):
                if h1 > h0:
                    vt.vt_kv_write_raw(st.kv, l, d, kc[h0 // g:h1 // g], vc[h0 // g:h1 // g])
        vt.vt_kv_set_length(st.kv, -1, wl.kv_len, stream)
        setup_s = time.perf_counter() - t_setup
        fused, why = vt.vt_decode_token_fused_available(st.part)
        xin = torch.from_numpy(wl.hidden(1).reshape(-1)).cuda()
        xout = torch.empty_like(xin)
        stream.synchronize()
        sch = TokenSchedule(vt, st, vt.vt_decode_token, xin, xout, stream, sched, wl.kv_len)
        ms = time_tokens(torch, sch, stream, steps, warmup)
        finite = bool(torch.isfinite(xout.float()).all().item())
        status = {"kv": vt.vt_kv_status(st.kv, clear=True), "partition": vt.vt_partition_status(st.part, clear=True)}
        del sch
    finally:
        torch.cuda.synchronize()
        st.close()
    hbm, _, _, peak_kind = measured_peaks()
    kv_mean = wl.kv_len + (min(steps, sched) - 1) / 2.0
    step_bytes = decode_bytes_per_token(wl, kv_mean) if bits == 16 else quant_bytes_per_token(wl, bits, kv_mean)
    achieved = step_bytes / (ms * 1e-3) / 1e9
    return {
        "workload": wl.name if bits == 16 else f"{wl.name}, every shard block-quantized to {bits} bits "
                                                f"(blocks of 32, fp16 scales)",
        "shape": f"{wl.n_layers} layers, D {wl.d_model}, {wl.n_heads} query / {wl.n_kv_heads} KV heads x "
                 f"{wl.d_head}, FFN {wl.d_ffn}; heads {[h1 - h0 for h0, h1 in wl.head_ranges]}, "
                 f"FFN columns {[c1 - c0 for c0, c1 in wl.ffn_ranges]}; KV {wl.kv_len} -> {wl.kv_len + sched - 1}",
        "value": round(1000.0 / ms, 3), "unit": "tok/s", "ms_per_step": round(ms, 5), "steps": steps,
        "token_kernel": "fused: one cooperative kernel per token" if fused else f"per-shard kernels ({why})",
        "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": hbm, "unit": "GB/s",
                     "frac": round(achieved / hbm, 4), "peak_kind": f"{peak_kind} copy bandwidth",
                     "bytes_per_launch": int(step_bytes)},
        "device_status": status, "finite": finite, "setup_s": round(setup_s, 1),
    }


# ------------------------------------------------------------------ shard latency sweep

def run_sweep(args):
    """Latency of one shard's decode step (vt_decode_step) against the shard's width (the 7B
    layer split n ways, n = 1, 2, 4, 8) and, for ATTN shards, the KV length: the measurements
    behind the planner's time model (a device's time for a shard = its bytes / a streaming rate).
    Each timed step is cold: the L2 is flushed (a 256 MB write) before it, and steps walk a stack
    of layers.  Fits time = t0 + bytes / rate over all points and feeds the fitted rate to
    vt_plan_layers for a 4-device plan of the 7B stack over a slow and a fast link."""
    import torch

    from paper_2607_07046_gb300 import build as vt_build
    from paper_2607_07046_gb300 import vt
    from paper_2607_07046_gb300.stack import Stack

    vt_build.build()
    torch.cuda.set_device(0)
    base = synthetic.WORKLOADS[2]
    layers = 4
    lengths = [128, 1024, 4096, 16384]
    cap = max(lengths) + 8
    flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
    D, dh, H, F = base.d_model, base.d_head, base.n_heads, base.d_ffn
    points = []
    for n in (1, 2, 4, 8):
        import dataclasses
        wl = dataclasses.replace(base, n_layers=layers, head_ranges=synthetic._even(H, n),
                                 ffn_ranges=synthetic._even(F, n))
        shapes = shapes_for(vt, wl, cap)
        with Stack(shapes, wl.layer_weights, wl.head_ranges, wl.ffn_ranges, cap) as st:
            x = torch.from_numpy(wl.hidden(1).reshape(-1)).cuda()
            out = torch.empty(D, dtype=torch.float32, device="cuda")
            hq, c = H // n, F // n
            w_attn = 2 * ((hq + 2 * hq) * dh * D + D * hq * dh)
            w_ffn = 2 * 3 * D * c

            def timed(fn, reps=12):
                ts = []
                for i in range(reps):
                    flush.zero_()
                    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                    e0.record()
                    fn(i % layers)
                    e1.record()
                    e1.synchronize()
                    ts.append(e0.elapsed_time(e1) * 1e3)
                return float(np.median(ts[2:]))

            for L in lengths:
                vt.vt_kv_set_length(st.kv, -1, L)
                us = timed(lambda l: vt.vt_decode_step(st.part, (l, 0, vt.VT_BLOCK_ATTN), x, st.kv, out))
                byt = w_attn + 2 * 2 * hq * dh * (L + 1)
                points.append({"block": "attn", "shards": n, "heads": hq, "kv_len": L, "us": round(us, 2),
                               "bytes": byt, "gbs": round(byt / us / 1e3, 1)})
            us = timed(lambda l: vt.vt_decode_step(st.part, (l, 0, vt.VT_BLOCK_FFN), x, None, out))
            points.append({"block": "ffn", "shards": n, "cols": c, "us": round(us, 2), "bytes": w_ffn,
                           "gbs": round(w_ffn / us / 1e3, 1)})
    # least-squares fit of time = t0 + bytes / rate
    A = np.array([[1.0, p["bytes"]] for p in points])
    y = np.array([p["us"] * 1e-6 for p in points])
    (t0, inv_rate), *_ = np.linalg.lstsq(A, y, rcond=None)
    rate = 1.0 / inv_rate
    sh = shapes_for(vt, base, base.kv_len + 8)
    plans = {}
    for name, link in (("wifi_60MBps", 60e6), ("nvlink_900GBps", 900e9)):
        pl, tot = vt.vt_plan_layers(sh, [rate] * 4, None, None, link, 2e-6, 1, base.kv_len)
        plans[name] = {"tp_blocks": sum(1 for b in pl if b["tp"]), "mp_blocks": sum(1 for b in pl if not b["tp"]),
                       "token_s": tot, "first_ffn": pl[1]["ranges"]}
    return {"sweep": "shard decode-step latency, 7B layer split n ways, cold L2", "points": points,
            "fit": {"t0_us": round(t0 * 1e6, 2), "rate_gbs": round(rate / 1e9, 1)},
            "plans_with_fitted_rate": plans}


# ------------------------------------------------------------------ reference arm (CPU oracle)

def run_reference(args):
    import oracle
    wl = synthetic.WORKLOADS[2]
    w = wl.layer_weights(0)
    L0 = wl.kv_len
    kc, vc = wl.kv_fill(0, L0, L0 + args.warmup + args.steps + 1)
    pos = L0
    for i in range(args.warmup):
        oracle.tp_layer(wl, w, wl.hidden(1, stream=600 + i), pos, kc, vc)
        pos += 1
    t0 = time.perf_counter()
    for i in range(args.steps):
        oracle.tp_layer(wl, w, wl.hidden(1, stream=700 + i), pos, kc, vc)
        pos += 1
    dt = (time.perf_counter() - t0) / max(args.steps, 1)
    per_token = dt * wl.n_layers
    value = 1.0 / per_token
    sample = (f"each step: one decode token through layer 0 of 32 (4-way TP shards, KV from {L0}), "
              f"timed; tok/s = 1 / (32 x step time), the x32 by layers stated in ms_per_token_extrapolated")
    return {"metric": METRIC, "value": round(value, 4), "unit": "tok/s", "n_gpus": 1,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(dt * 1e3, 3),
            "ms_per_token_extrapolated": round(per_token * 1e3, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "impl": "reference",
            "config": {"workload": WORKLOAD, "kv_len_start": L0, "partition": "heads 8/8/8/8, ffn 2752 x 4",
                       "implementation": "CPU oracle (fp64); a step is one layer of the token (timed), "
                                         "value extrapolated x32 by layers"},
            "cpu_baseline": {"value": round(value, 4), "unit": "tok/s", "cores": oracle.num_threads(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": round(value, 4), "unit": "tok/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=384)
    ap.add_argument("--warmup", type=int, default=8)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--prefill-steps", type=int, default=20,
                    help="timed 512-token prefills after the decode measurement (0: skip)")
    ap.add_argument("--sharded-steps", type=int, default=64,
                    help="timed tokens of the per-shard entry point, for context (0: skip)")
    ap.add_argument("--layers", type=int, default=0,
                    help="small case for profiling: only the first N layers of the stack")
    ap.add_argument("--sweep", action="store_true",
                    help="only the shard latency sweep (width x KV length) and the planner fed with its rate")
    ap.add_argument("--min-timed-s", type=float, default=0.3,
                    help="repeat the K-step timed region until it covers this many seconds in total")
    ap.add_argument("--other-steps", type=int, default=64,
                    help="timed tokens of the 13B and 8B decode workloads, 1 GPU only (0: skip)")
    ap.add_argument("--quantized", type=int, default=0, choices=[0, 4, 8],
                    help="only the 7B decode with every shard block-quantized to this many bits "
                         "(--other-steps timed tokens; --layers for a small case)")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    if args.sweep:
        print(json.dumps(run_sweep(args)), flush=True)
        return
    if args.quantized:
        print(json.dumps(run_decode_workload(2, max(args.other_steps, 1), args.warmup, args.quantized, args.layers)),
              flush=True)
        return
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(run_reference(args)), flush=True)
        return
    if world > 1:
        import torch
        torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", 0)))
        torch.distributed.init_process_group("nccl")
    line, clocks = run_decode(args, rank, world)
    line["clocks"] = clocks
    if world == 1 and args.other_steps > 0 and not args.layers:
        line["other_workloads"] = [run_decode_workload(cid, args.other_steps, 8) for cid in (3, 5)]
        line["quantized_shards"] = [run_decode_workload(2, args.other_steps, 8, bits) for bits in (8, 4)]
    if rank == 0 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline_decode(synthetic.WORKLOADS[2])
        if "prefill" in line:
            line["prefill"]["cpu_baseline"] = cpu_baseline_prefill(synthetic.WORKLOADS[4])
    if world > 1:
        import torch
        torch.distributed.barrier()
        torch.distributed.destroy_process_group()
    if rank == 0:
        print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
