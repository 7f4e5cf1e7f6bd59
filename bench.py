"""Benchmark of the AATC hot path on GB300: encode + decode attention over the packed cache.

Workload (default): the Llama-3.1-8B-shaped single layer -- 32 query heads, 8 kv-heads,
head_dim 128, batch 1, context 32768, 2.75 average bits.  One *step* = encode the full context
(32768 tokens x 8 kv-heads, K and V) into the packed cache, then 256 decode-attention steps with
random bf16 queries.  Inputs are synthetic (workloads/: seeded anisotropic Gaussian KV).

Reported metric (one JSON line): decode-attention GB/s on algorithmic packed-cache bytes
(codes + per-token scales, 96 B per token and kv-head at 2.75 bits) and its fraction of the
measured HBM copy bandwidth; encode Mtok/s alongside.  The packed cache is 25 MB, smaller than
L2, so the decodes rotate over 16 cache copies (403 MB > 129 MB L2).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
Under torchrun (N > 1) every rank runs the same workload on its own GPU (weak scaling; the
path has no data exchange); rank 0 prints the line.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import workloads as W  # noqa: E402

METRIC = "compressed-KV decode attn GB/s & % of HBM peak; encode Mtok/s (1 GB300)"
DECODE_KERNELS = "aatc_decode_fused_kernel + aatc_decode_merge_kernel"
DECODE_LAUNCHES_PER_CALL = 2
N_COPIES = 16
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "traffic.json")
PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    return ws, rank


def max_over_ranks(values, ws, device=None):
    """Each timing's maximum over the ranks (the slowest replica defines the job's time); a
    collective only when ws > 1 (any torch.distributed backend)."""
    import torch
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    if ws > 1:
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return [float(x) for x in t.cpu()]


def whole_job_rate(units_per_rank, ws, ms):
    """Weak scaling: every rank processes units_per_rank in the same (max-over-ranks) time."""
    return ws * units_per_rank / (ms * 1e-3)


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 50 ms during the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.out = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "50"], stdout=self.out,
                                         stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        return self

    def wait_first_sample(self, timeout_s: float = 3.0):
        """Block until nvidia-smi has written its first sample, so the timed region is covered."""
        if self.proc is None or not self.path:
            return
        t_end = time.time() + timeout_s
        while time.time() < t_end:
            self.out.flush()
            if os.path.getsize(self.path) > 0:
                return
            time.sleep(0.01)

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.out.close()

    def summary(self):
        if self.proc is None or not self.path:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


def _source_hash(path):
    with open(path, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


def _traffic(key):
    """DRAM bytes per launch of one measured kernel call from the committed ncu summaries
    (profiles/traffic.json), or None when the source it was taken on has changed since."""
    if not os.path.exists(TRAFFIC_FILE):
        return None
    with open(TRAFFIC_FILE) as f:
        d = json.load(f).get(key)
    if not d:
        return None
    src = os.path.join(ROOT, d["source"])
    if not os.path.exists(src) or d.get("source_sha256_16") != _source_hash(src):
        return None
    return d.get("bytes_per_call")


def build_case(aatc, cfg, avg_bits, device):
    ck, cv, cq = W.layer_calibration(cfg, 0)
    dm = aatc.dims(1, cfg.n_kv_heads, cfg.n_q_heads)
    p = aatc.calibrate(dm, ck[None], cv[None], cq[None], avg_bits)
    plan = aatc.Plan(dm, p["basis"], p["bits"], p["scales"])
    return plan, p


def decode_bytes(plan, cfg, batch, n_ctx):
    """Algorithmic bytes one decode reads: packed codes (sum of widths) + fp32 alpha, K and V."""
    bits = plan._bits.reshape(-1, 2, 128).astype(np.int64).sum(axis=2)      # (H_kv, 2) code bits per token
    per_token = float(np.sum(bits) / 8.0 + 4 * bits.size)
    return batch * n_ctx * per_token


# ------------------------------------------------------------------------------------ our arm

def sink_window_timing(aatc, plan, cfg, caches, kd, vd, qs, out, wspace, steps_dec):
    """Decode with the paper's full-precision sink (4) and recent window (128, step 16): coded
    tokens [4, 4 + n_coded) from the same packed caches plus 4 + n_window bf16 tokens, one
    softmax.  256 calls replayed as one CUDA graph, 5 replays; GB/s on packed + bf16 bytes."""
    import torch
    from paper_2608_14191_gb300.sink_window import SinkWindowState
    B, T = cfg.batch, cfg.n_ctx
    n_sink, n_coded, n_win = SinkWindowState(4, 128, 16).counts(T)
    idx = list(range(n_sink)) + list(range(n_sink + n_coded, T))
    kf, vf = kd[:, idx].contiguous(), vd[:, idx].contiguous()

    def calls():
        for i in range(steps_dec):
            aatc.decode_attention_sw(plan, 0, qs[i], caches[i % N_COPIES], n_sink, n_sink + n_coded, T, kf, vf,
                                     len(idx), out=out[i], workspace=wspace)
    for _ in range(2):
        calls()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        calls()
    g.replay()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(5):
        g.replay()
    e1.record()
    torch.cuda.synchronize()
    us = e0.elapsed_time(e1) * 1e3 / (5 * steps_dec)
    packed = decode_bytes(plan, cfg, B, n_coded)
    full = B * len(idx) * cfg.n_kv_heads * 2 * 128 * 2
    return {"us_per_call": round(us, 3), "gbs": round((packed + full) / (us * 1e-6) / 1e9, 2),
            "coded_tokens": n_coded, "full_precision_tokens": len(idx), "bytes_per_call": packed + full,
            "policy": "sink 4 + recent window 128 (step 16) in bf16, the rest coded"}


def sink_window_stream_timing(aatc, plan, cfg, kd, vd, qs, device, n_steps=256):
    """Token-by-token generation with the paper's sink / window policy on the Llama-shaped layer:
    the cache manager holds 32768 - 2 n_steps tokens (prefilled in one append), then n_steps
    untimed and n_steps timed steps of (append one token to every kv-head, decode attention).
    Appends write the new token in place; every 16th token flushes 16 window tokens through
    the encode.  Timed with CUDA events (device time of the whole loop, host dispatch included
    where the host is slower) and the host clock."""
    import torch
    from paper_2608_14191_gb300.sink_window import SinkWindowCache
    B, T = cfg.batch, cfg.n_ctx
    swc = SinkWindowCache(plan, 0, B, T, device)
    t0 = T - 2 * n_steps
    swc.append(kd[:, :t0], vd[:, :t0])
    out = torch.empty((B, cfg.n_q_heads, 128), dtype=torch.float32, device=device)
    ws = torch.empty(max(1, plan.workspace_bytes(B, T) // 4), dtype=torch.float32, device=device)
    stream = torch.cuda.current_stream()

    def steps(a):
        for t in range(a, a + n_steps):
            swc.append(kd[:, t:t + 1], vd[:, t:t + 1])
            swc.decode(qs[t % qs.shape[0]], out=out, workspace=ws)

    steps(t0)
    torch.cuda.synchronize()
    flushes0 = swc.state.n_coded
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    h0 = time.perf_counter()
    e0.record(stream)
    steps(t0 + n_steps)
    e1.record(stream)
    torch.cuda.synchronize()
    host_us = (time.perf_counter() - h0) * 1e6 / n_steps
    us = e0.elapsed_time(e1) * 1e3 / n_steps
    assert plan.device_error() == 0
    return {"us_per_token": round(us, 3), "host_us_per_token": round(host_us, 3),
            "tokens_flushed": swc.state.n_coded - flushes0, "block_relocations": swc.relocations,
            "what": f"{n_steps} steps of (append 1 token x {cfg.n_kv_heads} kv-heads, decode) at "
                    f"{T - n_steps} tokens, sink 4 + window 128 (step 16) kept in place"}


def hidden_encode_timing(aatc, device, d_model=4096, n_kv=8, n_q=32, n_tokens=32768, iters=10, warmup=3):
    """Encode straight from the layer input (Sec. 5 Step 1: the cache holds the coefficients of
    x A): Llama-3.1-8B-shaped layer input, d_model 4096, 8 kv-heads x K|V, 32768 tokens.  The
    plan is calibrated on K = X W of 4096 seeded hidden states and seeded projections; the
    kernel is a tensor-core GEMM (2 x 32768 x 4096 x 2048 flop) with the quantize / pack
    epilogue.  x is 268 MB (> L2), so back-to-back calls re-read it from HBM."""
    import torch
    seed = 1002
    x_cal = W.hidden_states(seed, 0, d_model, 4096)
    w_k = W.projection_weight(seed, 0, 0, d_model, n_kv)
    w_v = W.projection_weight(seed, 0, 1, d_model, n_kv)
    ck = (x_cal @ w_k).reshape(4096, n_kv, 128).transpose(1, 0, 2)[None]
    cv = (x_cal @ w_v).reshape(4096, n_kv, 128).transpose(1, 0, 2)[None]
    cfg = W.CONFIGS["llama_layer"]
    cq = np.stack([W.calibration_queries(cfg, 0, j) for j in range(n_q)])[None]
    dm = aatc.dims(1, n_kv, n_q)
    p = aatc.calibrate(dm, np.ascontiguousarray(ck), np.ascontiguousarray(cv), cq, 2.75)
    plan = aatc.Plan(dm, p["basis"], p["bits"], p["scales"])
    ah = aatc.hidden_operand(dm, w_k[None], w_v[None], p["basis"])
    a_hat = torch.from_numpy(ah.view(np.int16)).view(torch.bfloat16).to(device).contiguous()
    x = W.hidden_states_device(seed, 0, d_model, 1, n_tokens, device)
    cache = plan.new_cache(1, n_tokens, device)
    for _ in range(warmup):
        aatc.encode_hidden(plan, 0, x, a_hat, cache, 0, n_tokens)
    torch.cuda.synchronize()
    if iters == 0:
        assert plan.device_error() == 0
        plan.close()
        return {}
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(iters):
        aatc.encode_hidden(plan, 0, x, a_hat, cache, 0, n_tokens)
    e1.record()
    torch.cuda.synchronize()
    assert plan.device_error() == 0
    us = e0.elapsed_time(e1) * 1e3 / iters
    flop = 2.0 * n_tokens * d_model * n_kv * 2 * 128
    peaks = json.load(open(PEAKS_FILE)) if os.path.exists(PEAKS_FILE) else {}
    bf16 = float(peaks.get("bf16_tflops", 1900.0))
    tf = flop / (us * 1e-6) / 1e12
    plan.close()
    return {"us_per_call": round(us, 2), "mtok_s": round(n_tokens / us, 2), "tflops": round(tf, 1),
            "frac_of_measured_bf16": round(tf / bf16, 4),
            "workload": f"Llama-3.1-8B-shaped layer input: d_model {d_model}, {n_kv} kv-heads x K|V, "
                        f"{n_tokens} tokens, 2.75 bits"}


def stack_plan(aatc, cfg, avg_bits=2.75):
    """One plan for the whole stack with a separately calibrated basis, allocation and scales per
    layer and kv-head (each layer from its own seeded calibration set); layers are calibrated in
    parallel host threads (the planner call releases the GIL)."""
    import concurrent.futures as cf
    L, H = cfg.n_layers, cfg.n_kv_heads

    def one(layer):
        ck, cv, cq = W.layer_calibration(cfg, layer)
        return aatc.calibrate(aatc.dims(1, H, cfg.n_q_heads), ck[None], cv[None], cq[None], avg_bits)

    with cf.ThreadPoolExecutor(max_workers=min(16, os.cpu_count() or 4)) as ex:
        ps = list(ex.map(one, range(L)))
    basis = np.concatenate([p["basis"] for p in ps])
    bits = np.concatenate([p["bits"] for p in ps])
    scales = np.concatenate([p["scales"] for p in ps])
    return aatc.Plan(aatc.dims(L, H, cfg.n_q_heads), basis, bits, scales), bits


def stack_decode_timing(aatc, device, reps=10):
    """Decode through the Llama-3.1-8B-shaped 32-layer stack at 131072 tokens (one decode step =
    one call per layer, 101 MB of packed codes and alpha each, 3.2 GB in all, far above L2),
    timed as one CUDA graph of the 32 calls.  Every layer has its own calibrated plan (basis,
    widths and scales per kv-head) and its cache is encoded from its own synthetic K/V."""
    import torch
    cfg = W.CONFIGS["llama_stack"]
    n_layers, n_ctx = cfg.n_layers, cfg.n_ctx
    t0 = time.perf_counter()
    plan, bits = stack_plan(aatc, cfg)
    plan_s = time.perf_counter() - t0
    caches = []
    for layer in range(n_layers):
        kd, vd = W.kv_device(cfg, layer, 1, n_ctx, device)
        c = plan.new_cache(1, n_ctx, device)
        aatc.encode(plan, layer, kd, vd, c, 0, n_ctx)
        caches.append(c)
        del kd, vd
    q = W.queries_device(cfg, 0, 1, 1, device)[0]
    outs = torch.empty((n_layers, 1, cfg.n_q_heads, 128), dtype=torch.float32, device=device)
    ws = torch.empty(plan.workspace_bytes(1, n_ctx) // 4, dtype=torch.float32, device=device)

    def step():
        for layer in range(n_layers):
            aatc.decode_attention(plan, layer, q, caches[layer], n_ctx, n_ctx, out=outs[layer], workspace=ws)

    step()
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        step()
    for _ in range(3):
        graph.replay()
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(reps):
        graph.replay()
    e1.record(stream)
    torch.cuda.synchronize()
    assert plan.device_error() == 0
    us = e0.elapsed_time(e1) * 1e3 / (reps * n_layers)
    # bytes of one step: packed codes (each layer's widths / 8) + 4 B alpha per (token, kv-head, K|V)
    step_bytes = float(n_ctx * (np.sum(bits.astype(np.int64)) / 8.0 + 4 * n_layers * cfg.n_kv_heads * 2))
    nbytes = step_bytes / n_layers
    peak, kind = _peaks()
    gbs = nbytes / (us * 1e-6) / 1e9
    plan.close()
    return {"us_per_layer_call": round(us, 3), "gbs": round(gbs, 2), "bytes_per_call": nbytes,
            "frac_of_measured_hbm": round(gbs / peak, 4), "frac_of_nominal_8tbs": round(gbs / 8000.0, 4),
            "step_ms": round(us * n_layers / 1e3, 3), "plan_seconds": round(plan_s, 2),
            "roofline": {"bound": "hbm", "achieved": round(gbs, 2), "peak": peak, "unit": "GB/s",
                         "frac": round(gbs / peak, 4), "traffic": _traffic("decode_stack"),
                         "kernel": "one decode call (131072 tokens x 8 kv-heads)",
                         "peak_source": f"{kind} hbm_gbs (MEASURED_PEAKS.json)"},
            "workload": "Llama-3.1-8B-shaped stack: 32 layers x 131072 tokens x 8 kv-heads, one decode step "
                        "(32 calls in a CUDA graph), a separately calibrated plan per layer and kv-head"}


def qwen_timing(aatc, device, n_calls=64, reps=3, enc_iters=6, n_copies=4):
    """The Qwen-2.5-7B-shaped layer: prefill-encode of 16 sequences x 8192 tokens (28 query heads
    over 4 kv-heads, 268 MB of bf16 K/V input, > L2) as one encode call, then one batched decode
    step of all 16 sequences (G = 7, 50 MB of packed codes and alpha), timed as a CUDA graph of
    calls rotating over four packed-cache copies (201 MB > L2)."""
    import torch
    cfg = W.CONFIGS["qwen"]
    B, T = cfg.batch, cfg.n_ctx
    plan, _ = build_case(aatc, cfg, 2.75, device)
    kd, vd = W.kv_device(cfg, 0, B, T, device)
    qs = W.queries_device(cfg, 0, B, 4, device)
    caches = [plan.new_cache(B, T, device) for _ in range(n_copies)]
    stream = torch.cuda.current_stream()
    peak, kind = _peaks()
    ctr = [0]

    def enc():
        aatc.encode(plan, 0, kd, vd, caches[ctr[0] % n_copies], 0, T)
        ctr[0] += 1

    for _ in range(n_copies):
        enc()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(enc_iters):
        enc()
    e1.record(stream)
    torch.cuda.synchronize()
    enc_us = e0.elapsed_time(e1) * 1e3 / enc_iters
    in_bytes = (kd.numel() + vd.numel()) * 2
    out = torch.empty((B, cfg.n_q_heads, 128), dtype=torch.float32, device=device)
    ws = torch.empty(max(1, plan.workspace_bytes(B, T) // 4), dtype=torch.float32, device=device)

    def calls():
        for i in range(n_calls):
            aatc.decode_attention(plan, 0, qs[i % qs.shape[0]], caches[i % n_copies], T, T, out=out, workspace=ws)

    calls()
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        calls()
    graph.replay()
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(reps):
        graph.replay()
    e1.record(stream)
    torch.cuda.synchronize()
    assert plan.device_error() == 0
    dec_us = e0.elapsed_time(e1) * 1e3 / (reps * n_calls)
    dbytes = decode_bytes(plan, cfg, B, T)
    dec_gbs = dbytes / (dec_us * 1e-6) / 1e9
    enc_gbs = in_bytes / (enc_us * 1e-6) / 1e9
    plan.close()
    return {"workload": cfg.workload,
            "encode": {"us_per_call": round(enc_us, 2), "mtok_s": round(B * T / enc_us, 2),
                       "input_gbs": round(enc_gbs, 2), "frac_of_measured_hbm_on_input": round(enc_gbs / peak, 4),
                       "frac_of_nominal_8tbs": round(enc_gbs / 8000.0, 4), "input_bytes": in_bytes},
            "decode": {"us_per_call": round(dec_us, 3), "gbs": round(dec_gbs, 2), "bytes_per_call": dbytes,
                       "frac_of_measured_hbm": round(dec_gbs / peak, 4),
                       "frac_of_nominal_8tbs": round(dec_gbs / 8000.0, 4),
                       "mtok_s": round(B * T / dec_us, 2)},
            "roofline": {"bound": "hbm", "achieved": round(dec_gbs, 2), "peak": peak, "unit": "GB/s",
                         "frac": round(dec_gbs / peak, 4), "traffic": _traffic("decode_qwen"),
                         "kernel": "one batched decode call (16 x 8192 tokens x 4 kv-heads, G = 7)",
                         "peak_source": f"{kind} hbm_gbs (MEASURED_PEAKS.json)"},
            "timing": f"encode: {enc_iters} calls rotating over {n_copies} caches; decode: {n_calls}-call CUDA graph "
                      f"x {reps} over {n_copies} packed-cache copies"}


def group_plan_for(aatc, cfg, g_h, avg_bits=2.75):
    """Head-group plan of layer 0 of `cfg` from the host group planner (one call per (group,
    kind) stream, run on host threads at once); returns (plan, seconds)."""
    import concurrent.futures as cf
    H, G = cfg.n_kv_heads, cfg.group
    ng, n = H // g_h, 128 * g_h
    ck, cv, cq = W.layer_calibration(cfg, 0)
    jobs = []
    for g in range(ng):
        hk = slice(g * g_h, (g + 1) * g_h)
        jobs.append((g, 0, ck[hk], cq[g * g_h * G:(g + 1) * g_h * G]))
        jobs.append((g, 1, cv[hk], None))
    basis = np.zeros((1, ng, 2, n, n), np.float32)
    bits = np.zeros((1, ng, 2, n), np.uint8)
    scales = np.ones((1, ng, 2, n), np.float32)
    t0 = time.time()
    with cf.ThreadPoolExecutor(max_workers=len(jobs)) as ex:
        res = list(ex.map(lambda j: aatc.calibrate_head_group(j[2], j[3], avg_bits, group=G), jobs))
    for (g, kind, _, _), p in zip(jobs, res):
        basis[0, g, kind], bits[0, g, kind], scales[0, g, kind] = p["basis"], p["bits"], p["scales"]
    plan = aatc.GroupPlan(aatc.dims(1, H, cfg.n_q_heads), g_h, basis, bits, scales)
    return plan, time.time() - t0


def group_timing(aatc, device, g_h=4, n_calls=64, reps=3, enc_iters=6, n_copies=16):
    """Head-group bases on the Llama-shaped layer (Sec. 5 Step 1 with the paper's Llama grouping:
    two groups of four kv-heads, 512 channels per group stream): encode of 32768 tokens and the
    decode of all 32 query heads, timed like the headline (decode calls as one CUDA graph over
    packed-cache copies larger than L2)."""
    import torch
    cfg = W.CONFIGS["llama_layer"]
    B, T = 1, cfg.n_ctx
    plan, plan_s = group_plan_for(aatc, cfg, g_h)
    kd, vd = W.kv_device(cfg, 0, B, T, device)
    qs = W.queries_device(cfg, 0, B, 8, device)
    caches = [plan.new_cache(B, T, device) for _ in range(n_copies)]
    stream = torch.cuda.current_stream()
    peak, kind = _peaks()
    ctr = [0]

    def enc():
        aatc.encode(plan, 0, kd, vd, caches[ctr[0] % n_copies], 0, T)
        ctr[0] += 1

    for _ in range(n_copies):
        enc()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(enc_iters):
        enc()
    e1.record(stream)
    torch.cuda.synchronize()
    enc_us = e0.elapsed_time(e1) * 1e3 / enc_iters
    in_bytes = (kd.numel() + vd.numel()) * 2
    out = torch.empty((B, cfg.n_q_heads, 128), dtype=torch.float32, device=device)
    ws = torch.empty(max(1, plan.workspace_bytes(B, T) // 4), dtype=torch.float32, device=device)

    def calls():
        for i in range(n_calls):
            aatc.decode_attention(plan, 0, qs[i % qs.shape[0]], caches[i % n_copies], T, T, out=out, workspace=ws)

    calls()
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        calls()
    graph.replay()
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(reps):
        graph.replay()
    e1.record(stream)
    torch.cuda.synchronize()
    assert plan.device_error() == 0
    dec_us = e0.elapsed_time(e1) * 1e3 / (reps * n_calls)
    # algorithmic bytes: the packed codes (sum of widths) and one fp32 alpha per group stream
    ng = cfg.n_kv_heads // g_h
    dbytes = float(B * T * (plan._bits.astype(np.int64).sum() / 8.0 + 4 * ng * 2))
    dec_gbs = dbytes / (dec_us * 1e-6) / 1e9
    enc_gbs = in_bytes / (enc_us * 1e-6) / 1e9
    res = {"workload": f"Llama-3.1-8B-shaped layer with head-group bases: 2 groups x {g_h} kv-heads "
                       f"({128 * g_h} channels per group stream), {T} tokens, 32 query heads, 2.75 bits",
           "encode": {"us_per_call": round(enc_us, 2), "input_gbs": round(enc_gbs, 2),
                      "frac_of_measured_hbm_on_input": round(enc_gbs / peak, 4)},
           "decode": {"us_per_call": round(dec_us, 3), "gbs": round(dec_gbs, 2), "bytes_per_call": dbytes,
                      "frac_of_measured_hbm": round(dec_gbs / peak, 4),
                      "workspace_bytes": plan.workspace_bytes(B, T)},
           "roofline": {"bound": "hbm", "achieved": round(dec_gbs, 2), "peak": peak, "unit": "GB/s",
                        "frac": round(dec_gbs / peak, 4), "traffic": _traffic("decode_groups"),
                        "kernel": "one group decode call (query + digit attention + merge kernels)",
                        "peak_source": f"{kind} hbm_gbs (MEASURED_PEAKS.json)"},
           "planner_seconds": round(plan_s, 2),
           "timing": f"encode: {enc_iters} calls rotating over {n_copies} caches; decode: {n_calls}-call CUDA graph "
                     f"x {reps} over {n_copies} packed-cache copies"}
    plan.close()
    return res


def bf16_decode_timing(aatc, kd, vd, qs, n_ctx, packed_us, n_calls=64, reps=3):
    """The uncompressed reference decode (split-K attention over the bf16 K/V with the same shapes
    and queries), timed like the packed decode: a CUDA graph of calls alternating two K/V copies
    (2 x 134 MB > L2).  GB/s on the bf16 bytes a call reads, and the packed decode's speed-up
    over it (the byte ratio 512 / 96 = 5.3 bounds it at 2.75 bits)."""
    import torch
    pairs = [(kd, vd), (kd.clone(), vd.clone())]
    batch, n_kv, n_q = kd.shape[0], kd.shape[2], qs.shape[2]
    out = torch.empty((batch, n_q, 128), dtype=torch.float32, device=kd.device)
    ws = torch.empty(max(1, aatc.bf16_workspace_bytes(batch, n_kv, n_q, n_ctx) // 4), dtype=torch.float32,
                     device=kd.device)

    def calls():
        for i in range(n_calls):
            k_, v_ = pairs[i & 1]
            aatc.bf16_decode_attention(k_, v_, qs[i % qs.shape[0]], n_ctx, out=out, workspace=ws)

    calls()
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        calls()
    graph.replay()
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(reps):
        graph.replay()
    e1.record(stream)
    torch.cuda.synchronize()
    us = e0.elapsed_time(e1) * 1e3 / (reps * n_calls)
    nbytes = (kd.numel() + vd.numel()) * 2
    peak, _ = _peaks()
    return {"us_per_call": round(us, 3), "gbs": round(nbytes / (us * 1e-6) / 1e9, 2), "bytes_per_call": nbytes,
            "frac_of_measured_hbm": round(nbytes / (us * 1e-6) / 1e9 / peak, 4),
            "packed_speedup": round(us / packed_us, 3),
            "what": "uncompressed bf16 K/V reference decode, same shapes and queries, 64 calls per CUDA graph"}


def prefill_timing(aatc, device, iters=2, batch=None, reference=True):
    """Prefill attention over the packed cache on the Qwen-2.5-7B-shaped layer: 16 sequences x
    8192 tokens, 28 query heads over 4 kv-heads, causal (the chunk is the whole context, encoded
    first).  Flop = 2 (QK) + 2 (PV) x 128 x 28 heads x 16 x 8192 x 8193 / 2 causal pairs.  For
    context, the same attention on the uncompressed bf16 K/V by torch's scaled_dot_product_attention
    (a library kernel, not this path)."""
    import torch
    cfg = W.CONFIGS["qwen"]
    B, T = cfg.batch if batch is None else batch, cfg.n_ctx
    plan, _ = build_case(aatc, cfg, 2.75, device)
    kd, vd = W.kv_device(cfg, 0, B, T, device)
    cache = plan.new_cache(B, T, device)
    aatc.encode(plan, 0, kd, vd, cache, 0, T)
    gen = torch.Generator(device=device)
    gen.manual_seed(W.torch_seed(cfg.seed, 0, 0, 0, "query"))
    q = torch.randn((B, T, cfg.n_q_heads, 128), generator=gen, device=device).to(torch.bfloat16)
    out = torch.empty((B, T, cfg.n_q_heads, 128), dtype=torch.float32, device=device)
    aatc.prefill_attention(plan, 0, q, 0, cache, T, T, out=out)
    torch.cuda.synchronize()
    if iters == 0:
        assert plan.device_error() == 0
        plan.close()
        return {}
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(iters):
        aatc.prefill_attention(plan, 0, q, 0, cache, T, T, out=out)
    e1.record()
    torch.cuda.synchronize()
    assert plan.device_error() == 0
    ms = e0.elapsed_time(e1) / iters
    flop = 4.0 * 128 * cfg.n_q_heads * B * T * (T + 1) / 2
    # uncompressed bf16 reference (library SDPA), same shapes, causal, GQA by repeating kv-heads
    g = cfg.n_q_heads // cfg.n_kv_heads
    qt = q.transpose(1, 2)
    kt = kd.transpose(1, 2).repeat_interleave(g, dim=1)
    vt = vd.transpose(1, 2).repeat_interleave(g, dim=1)
    torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, is_causal=True)
    torch.cuda.synchronize()
    e0.record()
    for _ in range(iters):
        torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, is_causal=True)
    e1.record()
    torch.cuda.synchronize()
    ms_ref = e0.elapsed_time(e1) / iters
    peaks = json.load(open(PEAKS_FILE)) if os.path.exists(PEAKS_FILE) else {}
    bf16 = float(peaks.get("bf16_tflops", 1900.0))
    tf = flop / (ms * 1e-3) / 1e12
    plan.close()
    return {"ms_per_call": round(ms, 3), "tflops": round(tf, 1), "frac_of_measured_bf16": round(tf / bf16, 4),
            "bf16_sdpa_ms_uncompressed": round(ms_ref, 3),
            "workload": f"Qwen-2.5-7B-shaped layer: {B} x {T} tokens, {cfg.n_q_heads}/{cfg.n_kv_heads} heads, "
                        f"causal prefill over the packed cache (2.75 bits)"}


def sweep_timing(aatc, device, n_calls=32, reps=3, enc_iters=6):
    """Bit-budget sweep on the Llama shape at batch 4 x 32768 tokens: per budget (1.5 / 2 / 2.75 /
    4 bits) a plan, the encode of all K/V (536.9 MB of bf16 input, > L2) and the decode (a CUDA
    graph of calls alternating two packed-cache copies), against the bf16 reference decode of the
    same K/V and queries.  The speed-up is bounded by the byte ratio 512 / (sum b / 8 + 4)."""
    import torch
    cfg = W.CONFIGS["sweep"]
    B, T = cfg.batch, cfg.n_ctx
    kd, vd = W.kv_device(cfg, 0, B, T, device)
    qs = W.queries_device(cfg, 0, B, 4, device)
    stream = torch.cuda.current_stream()
    peak, _ = _peaks()
    ref = bf16_decode_timing(aatc, kd, vd, qs, T, 1.0, n_calls=n_calls, reps=reps)
    in_bytes = (kd.numel() + vd.numel()) * 2

    def timed(fn, iters):
        fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(iters):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) * 1e3 / iters              # us per iteration

    rows = []
    for bits in cfg.avg_bits:
        plan, _ = build_case(aatc, cfg, bits, device)
        caches = [plan.new_cache(B, T, device) for _ in range(2)]
        ctr = [0]

        def enc():
            aatc.encode(plan, 0, kd, vd, caches[ctr[0] & 1], 0, T)
            ctr[0] += 1

        enc_us = timed(enc, enc_iters)
        for c in caches:
            aatc.encode(plan, 0, kd, vd, c, 0, T)
        out = torch.empty((B, cfg.n_q_heads, 128), dtype=torch.float32, device=device)
        ws = torch.empty(max(1, plan.workspace_bytes(B, T) // 4), dtype=torch.float32, device=device)

        def calls():
            for i in range(n_calls):
                aatc.decode_attention(plan, 0, qs[i % qs.shape[0]], caches[i & 1], T, T, out=out, workspace=ws)

        calls()
        torch.cuda.synchronize()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            calls()
        dec_us = timed(graph.replay, reps) / n_calls
        nbytes = decode_bytes(plan, cfg, B, T)
        per_token = nbytes / (B * T * cfg.n_kv_heads)
        rows.append({"avg_bits": bits, "bytes_per_token_kvhead": per_token,
                     "encode_us": round(enc_us, 2), "encode_mtok_s": round(B * T / enc_us, 2),
                     "encode_input_gbs": round(in_bytes / (enc_us * 1e-6) / 1e9, 2),
                     "decode_us": round(dec_us, 3), "decode_gbs": round(nbytes / (dec_us * 1e-6) / 1e9, 2),
                     "decode_frac_of_measured_hbm": round(nbytes / (dec_us * 1e-6) / 1e9 / peak, 4),
                     "speedup_vs_bf16": round(ref["us_per_call"] / dec_us, 3),
                     "byte_ratio_vs_bf16": round(512.0 / per_token, 3)})
        del graph
        plan.close()
    return {"workload": cfg.workload, "bf16_decode_us": ref["us_per_call"], "bf16_decode_gbs": ref["gbs"],
            "budgets": rows,
            "timing": f"encode: {enc_iters} calls alternating two caches; decode: {n_calls}-call CUDA graph x {reps}, "
                      "two packed-cache copies alternating; bf16: two K/V copies alternating (537 MB each)"}


def planner_timing(aatc):
    """Host planner rows: the global cross-layer allocation on Llama-3.1-8B-shaped statistics
    (32 layers x 8 kv-heads x K|V x 128 channels; seeded log-normal spectra), median of 5 runs."""
    rng = np.random.default_rng(1004)
    L, H = 32, 8
    s2 = -np.sort(-rng.lognormal(0.0, 1.5, (L, H, 2, 128)), axis=-1)
    w = np.ones_like(s2)
    dm = aatc.dims(L, H, 32)
    ts = []
    for _ in range(5):
        t0 = time.perf_counter()
        aatc.allocate_global(dm, s2, w, 2.75, 2.75, n_protect=3)
        ts.append(time.perf_counter() - t0)
    return {"global_allocation_ms": round(1e3 * float(np.median(ts)), 3),
            "shape": "32 layers x 8 kv-heads x K|V x 128 channels, 2.75 bits, first 3 layers protected"}


def run_ours(args):
    import torch
    import paper_2608_14191_gb300 as aatc
    from paper_2608_14191_gb300 import build as bld

    ws_, rank = _dist()
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if ws_ > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    if rank == 0 or not os.path.exists(bld.LIB):
        bld.build()
    if ws_ > 1:
        torch.distributed.barrier()
    aatc.load()

    cfg = W.CONFIGS[args.config]
    avg_bits = cfg.avg_bits[-1] if args.bits is None else args.bits
    B, T, steps_dec = cfg.batch, cfg.n_ctx, cfg.decode_steps
    plan, params = build_case(aatc, cfg, avg_bits, dev)
    kd, vd = W.kv_device(cfg, 0, B, T, dev)
    qs = W.queries_device(cfg, 0, B, steps_dec, dev)
    caches = [plan.new_cache(B, T, dev) for _ in range(N_COPIES)]
    for c in caches:
        aatc.encode(plan, 0, kd, vd, c, 0, T)
    out = torch.empty((steps_dec, B, cfg.n_q_heads, 128), dtype=torch.float32, device=dev)
    wsb = plan.workspace_bytes(B, T)
    wspace = torch.empty(wsb // 4, dtype=torch.float32, device=dev)
    torch.cuda.synchronize()

    def decodes(step):
        for i in range(steps_dec):
            aatc.decode_attention(plan, 0, qs[i], caches[(step * steps_dec + i) % N_COPIES], T, T, out=out[i],
                                  workspace=wspace)

    # CUDA graphs of the 256 decode calls, one per rotation offset (a step's decodes start at
    # copy (step * 256) % 16 = 0, so one graph serves every step)
    for _ in range(2):
        decodes(0)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        decodes(0)
    torch.cuda.synchronize()

    stream = torch.cuda.current_stream()
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]

    def step_dev(s, e3=None):
        if e3:
            e3[0].record(stream)
        aatc.encode(plan, 0, kd, vd, caches[s % N_COPIES], 0, T)
        if e3:
            e3[1].record(stream)
        graph.replay()
        if e3:
            e3[2].record(stream)

    for s in range(args.warmup):
        step_dev(s)
    torch.cuda.synchronize()
    if ws_ > 1:
        torch.distributed.barrier()
    with ClockSampler(local) as clk:
        clk.wait_first_sample()
        step_dev(0)                                  # untimed: clocks back up after the wait
        torch.cuda.synchronize()
        t_start = torch.cuda.Event(enable_timing=True)
        t_end = torch.cuda.Event(enable_timing=True)
        t_start.record(stream)
        for s in range(args.steps):
            step_dev(s, ev[s])
        t_end.record(stream)
        torch.cuda.synchronize()
    if ws_ > 1:
        torch.distributed.barrier()
    total_ms = t_start.elapsed_time(t_end)
    enc_ms = [e[0].elapsed_time(e[1]) for e in ev]
    dec_ms = [e[1].elapsed_time(e[2]) for e in ev]
    clocks = clk.summary()

    # end to end through the public API from pinned host buffers (no graphs), as a serving loop
    # runs it: the inputs of step s + 1 are copied in on a second stream while step s computes,
    # and step s's outputs are read back on that stream once its decodes are done (two device
    # sets of inputs and outputs).  Every step's host <-> device copies are inside the timed region.
    kh = torch.empty(kd.shape, dtype=torch.bfloat16, pin_memory=True)
    vh = torch.empty(vd.shape, dtype=torch.bfloat16, pin_memory=True)
    qh = torch.empty(qs.shape, dtype=torch.bfloat16, pin_memory=True)
    oh = [torch.empty(out.shape, dtype=torch.float32, pin_memory=True) for _ in range(2)]
    kh.copy_(kd)
    vh.copy_(vd)
    qh.copy_(qs)
    kdd = [torch.empty_like(kd) for _ in range(2)]
    vdd = [torch.empty_like(vd) for _ in range(2)]
    qsd = [torch.empty_like(qs) for _ in range(2)]
    outd = [torch.empty_like(out) for _ in range(2)]
    copy_stream = torch.cuda.Stream()
    ev_in = [torch.cuda.Event() for _ in range(2)]       # inputs of set j are on the device
    ev_done = [torch.cuda.Event() for _ in range(2)]     # compute on set j finished
    ev_out = [torch.cuda.Event() for _ in range(2)]      # outputs of set j are on the host
    recorded = {"done": [False, False], "out": [False, False]}

    def h2d(j):
        with torch.cuda.stream(copy_stream):
            if recorded["done"][j]:
                copy_stream.wait_event(ev_done[j])        # the last step on set j consumed its inputs
            kdd[j].copy_(kh, non_blocking=True)
            vdd[j].copy_(vh, non_blocking=True)
            qsd[j].copy_(qh, non_blocking=True)
            ev_in[j].record(copy_stream)

    def compute(s):
        j = s & 1
        stream.wait_event(ev_in[j])
        if recorded["out"][j]:
            stream.wait_event(ev_out[j])                  # outd[j] has been read back
        aatc.encode(plan, 0, kdd[j], vdd[j], caches[s % N_COPIES], 0, T)
        for i in range(steps_dec):
            aatc.decode_attention(plan, 0, qsd[j][i], caches[(s * steps_dec + i) % N_COPIES], T, T, out=outd[j][i],
                                  workspace=wspace)
        ev_done[j].record(stream)
        recorded["done"][j] = True
        with torch.cuda.stream(copy_stream):
            copy_stream.wait_event(ev_done[j])
            oh[j].copy_(outd[j], non_blocking=True)
            ev_out[j].record(copy_stream)
        recorded["out"][j] = True

    def run_e2e(n):
        h2d(0)
        for s in range(n):
            if s + 1 < n:
                h2d((s + 1) & 1)
            compute(s)
        stream.wait_event(ev_out[(n - 1) & 1])          # the last read-back ends the region

    e2e_steps = max(2, min(args.steps, 10))
    run_e2e(2)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    copy_stream.wait_stream(stream)                      # the first copy starts inside the region
    run_e2e(e2e_steps)
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = e0.elapsed_time(e1) / e2e_steps
    h2d = kd.numel() * 2 + vd.numel() * 2 + qs.numel() * 2
    d2h = out.numel() * 4
    assert plan.device_error() == 0

    # max over ranks, then only rank 0 goes on (the context legs below are single-GPU figures)
    total_ms, dec_mean, enc_mean, e2e_ms = max_over_ranks(
        [total_ms, float(np.mean(dec_ms)), float(np.mean(enc_ms)), e2e_ms], ws_, device=dev)
    if ws_ > 1:
        torch.distributed.destroy_process_group()
    if rank != 0:
        return

    sw = sink_window_timing(aatc, plan, cfg, caches, kd, vd, qs, out, wspace, steps_dec)
    sw["streaming"] = sink_window_stream_timing(aatc, plan, cfg, kd, vd, qs, dev)
    ref16 = bf16_decode_timing(aatc, kd, vd, qs, T, dec_mean / steps_dec * 1e3)
    qwen = qwen_timing(aatc, dev)
    groups = group_timing(aatc, dev)
    stack = stack_decode_timing(aatc, dev)
    hid = hidden_encode_timing(aatc, dev)
    pre = prefill_timing(aatc, dev)
    sweep = sweep_timing(aatc, dev)

    peak, peak_kind = _peaks()
    dbytes = decode_bytes(plan, cfg, B, T)
    per_decode_ms = dec_mean / steps_dec
    gbs = whole_job_rate(dbytes, ws_, per_decode_ms) / 1e9      # whole job
    achieved = dbytes / (per_decode_ms * 1e-3) / 1e9              # per launch (one GPU)
    enc_tokens = B * T
    enc_in_bytes = B * T * cfg.n_kv_heads * 2 * 128 * 2
    line = {
        "metric": METRIC,
        "value": round(gbs, 2),
        "unit": "GB/s",
        "n_gpus": ws_,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(total_ms / args.steps, 4),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f32",
        "data": "synthetic (seeded anisotropic Gaussian KV, power-law spectrum, key outliers; bf16)",
        "config": {"workload": cfg.workload, "avg_bits": avg_bits, "batch": B, "n_ctx": T,
                   "n_kv_heads": cfg.n_kv_heads, "n_q_heads": cfg.n_q_heads, "decode_steps_per_step": steps_dec,
                   "l2": f"decodes rotate over {N_COPIES} packed-cache copies "
                         f"({N_COPIES * dbytes / 1e6:.0f} MB > 129 MB L2); encode input {enc_in_bytes / 1e6:.0f} MB",
                   "parallelism": f"replica x{ws_}", "decode_graph": "256 decode calls replayed as one CUDA graph"},
        "decode": {"gbs": round(achieved, 2), "us_per_call": round(per_decode_ms * 1e3, 3),
                   "bytes_per_call": dbytes, "frac_of_measured_hbm": round(achieved / peak, 4),
                   "frac_of_nominal_8tbs": round(achieved / 8000.0, 4)},
        "encode": {"mtok_s": round(ws_ * enc_tokens / (enc_mean * 1e-3) / 1e6, 2),
                   "us_per_call": round(enc_mean * 1e3, 2),
                   "input_gbs": round(enc_in_bytes / (enc_mean * 1e-3) / 1e9, 2),
                   "frac_of_measured_hbm_on_input": round(enc_in_bytes / (enc_mean * 1e-3) / 1e9 / peak, 4)},
        "roofline": {"bound": "hbm", "achieved": round(achieved, 2), "peak": peak, "unit": "GB/s",
                     "frac": round(achieved / peak, 4), "traffic": _traffic("decode_layer"),
                     "kernel": DECODE_KERNELS + " (one decode call)",
                     "peak_source": f"{peak_kind} hbm_gbs (MEASURED_PEAKS.json)"},
        "roofline_encode": {"bound": "hbm", "achieved": round(enc_in_bytes / (enc_mean * 1e-3) / 1e9, 2),
                            "peak": peak, "unit": "GB/s",
                            "frac": round(enc_in_bytes / (enc_mean * 1e-3) / 1e9 / peak, 4),
                            "traffic": _traffic("encode_layer"), "algorithmic_bytes": enc_in_bytes,
                            "kernel": "aatc_encode_kernel (one encode of the layer: bf16 K/V input bytes)",
                            "peak_source": f"{peak_kind} hbm_gbs (MEASURED_PEAKS.json)"},
        "e2e": {"value": round(ws_ * steps_dec * dbytes / (e2e_ms * 1e-3) / 1e9, 2), "unit": "GB/s",
                "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
                "ms_per_step": round(e2e_ms, 4),
                "what": "per step: H2D of K, V and queries from pinned host memory, encode, 256 decode calls "
                        "through the public API, D2H of all outputs; the next step's H2D and this step's "
                        "D2H run on a second stream, overlapping compute"},
        "gpu_launches": args.steps * (1 + DECODE_LAUNCHES_PER_CALL * steps_dec),
        "clocks": clocks,
        "planner": planner_timing(aatc),
        "sink_window": sw,
        "bf16_decode": ref16,
        "qwen_layer": qwen,
        "head_groups": groups,
        "decode_llama_stack": stack,
        "encode_hidden": hid,
        "prefill": pre,
        "sweep": sweep,
    }
    if not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(cfg, avg_bits, budget_s=args.cpu_seconds,
                                            all_cores_s=min(10.0, args.cpu_seconds))
        line["cpu_baseline"]["oracle_encode_and_planner"] = oracle_encode_timing(cfg, avg_bits)
        line["cpu_baseline"]["code_agreement"] = oracle_code_agreement(params, caches[0], kd, vd, cfg, plan.n_words)
    print(json.dumps(line), flush=True)
    if ws_ > 1:
        torch.distributed.destroy_process_group()


# ------------------------------------------------------------------------------ oracle baseline

_ORACLE_CHILD = r"""
import json, os, sys, time
import numpy as np
sys.path.insert(0, sys.argv[1])
from oracle import aatc_oracle as O
d = np.load(sys.argv[2])
budget = float(sys.argv[3])
g = int(d["group"]); hkv = int(d["hkv"])
t0 = time.perf_counter(); n_done = 0; bytes_done = 0.0
while True:
    for h in range(hkv):
        hh = []
        for kind in (0, 1):
            bits = d["bits"][h, kind].astype(np.int64)
            codes = O.unpack_records(d["records"][h, kind], bits)
            hh.append(O.dequantize_f32(codes, d["alpha"][h, kind], d["scales"][h, kind], bits))
        O.decode_attention(d["q"][h * g:(h + 1) * g], hh[0][None], hh[1][None], d["basis"][h, 0][None],
                           d["basis"][h, 1][None], g)
    n_done += 1
    bytes_done += float(d["bytes"])
    if time.perf_counter() - t0 > budget:
        break
el = time.perf_counter() - t0
print(json.dumps({"seconds": el, "decodes": n_done, "bytes": bytes_done}))
"""


def oracle_sample(cfg, avg_bits, n_tokens):
    """CPU-only input for the oracle: its own plan (from the library's numpy twin: the oracle
    planner) and its own encode of n_tokens per stream."""
    from oracle import aatc_oracle as O
    ck, cv, cq = W.layer_calibration(cfg, 0)
    k, v = W.kv_host(cfg, 0, 1, n_tokens)
    g = cfg.group
    H = cfg.n_kv_heads
    recs, alphas, bits_all, scales_all, basis_all = [], [], [], [], []
    for h in range(H):
        rr, aa, bb, ss, uu = [], [], [], [], []
        for kind, x, cal in ((0, k, ck), (1, v, cv)):
            qsh = [cq[j].astype(np.float64) for j in range(h * g, (h + 1) * g)] if kind == 0 else None
            p = O.plan_stream(cal[h].astype(np.float64), avg_bits, queries_by_head=qsh)
            ub = W.to_bf16(p["basis"]).astype(np.float64)
            codes, alpha, _ = O.encode_stream(x[0, :, h, :].astype(np.float64), ub, p["bits"], p["scales"])
            nw = O.record_words([p["bits"]])
            rr.append(O.pack_records(codes, p["bits"], nw))
            aa.append(alpha.astype(np.float32))
            bb.append(p["bits"])
            ss.append(p["scales"].astype(np.float32))
            uu.append(p["basis"].astype(np.float32))
        nw = max(r.shape[1] for r in rr)
        rr = [np.pad(r, ((0, 0), (0, nw - r.shape[1]))) for r in rr]
        recs.append(rr)
        alphas.append(aa)
        bits_all.append(bb)
        scales_all.append(ss)
        basis_all.append(uu)
    q = W.queries_host(cfg, 0, 1, 1)[0, 0]
    bits_arr = np.array(bits_all)
    per_token = float(np.sum(bits_arr) / 8.0 + 4 * H * 2)
    return {"records": np.array(recs), "alpha": np.array(alphas), "bits": bits_arr,
            "scales": np.array(scales_all), "basis": np.array(basis_all), "q": q, "group": g, "hkv": H,
            "bytes": per_token * n_tokens}


def _run_oracle_children(path, budget_s, n_proc):
    """n_proc single-threaded oracle processes over the same sample at once (exec'd children, no
    fork of this process's CUDA state); returns summed decodes and bytes and the longest time."""
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")
    procs = [subprocess.Popen([sys.executable, "-c", _ORACLE_CHILD, ROOT, path, str(budget_s)],
                              stdout=subprocess.PIPE, stderr=subprocess.PIPE, text=True, env=env)
             for _ in range(n_proc)]
    out = {"seconds": 0.0, "decodes": 0, "bytes": 0.0}
    err = None
    for pr in procs:
        so, se = pr.communicate(timeout=600)
        if pr.returncode != 0:
            err = se[-300:]
            continue
        res = json.loads(so.strip().splitlines()[-1])
        out["seconds"] = max(out["seconds"], res["seconds"])
        out["decodes"] += res["decodes"]
        out["bytes"] += res["bytes"]
    return out, err


_ORACLE_ENCODE_CHILD = r"""
import json, sys, time
import numpy as np
sys.path.insert(0, sys.argv[1])
from oracle import aatc_oracle as O
import workloads as W
cfg = W.CONFIGS[sys.argv[2]]
avg_bits = float(sys.argv[3]); n_tok = int(sys.argv[4]); budget = float(sys.argv[5])
ck, cv, cq = W.layer_calibration(cfg, 0)
k, v = W.kv_host(cfg, 0, 1, n_tok)
g = cfg.group
t0 = time.perf_counter()
plans = []
for h in range(cfg.n_kv_heads):
    for kind, cal in ((0, ck), (1, cv)):
        qsh = [cq[j].astype(np.float64) for j in range(h * g, (h + 1) * g)] if kind == 0 else None
        plans.append(O.plan_stream(cal[h].astype(np.float64), avg_bits, queries_by_head=qsh))
plan_s = time.perf_counter() - t0
t0 = time.perf_counter(); reps = 0
while True:
    i = 0
    for h in range(cfg.n_kv_heads):
        for kind, x in ((0, k), (1, v)):
            p = plans[i]; i += 1
            ub = W.to_bf16(p["basis"]).astype(np.float64)
            codes, alpha, _ = O.encode_stream(x[0, :, h, :].astype(np.float64), ub, p["bits"], p["scales"])
            O.pack_records(codes, p["bits"], O.record_words([p["bits"]]))
    reps += 1
    if time.perf_counter() - t0 > budget:
        break
print(json.dumps({"plan_seconds": plan_s, "encode_seconds": time.perf_counter() - t0, "reps": reps}))
"""


def oracle_encode_timing(cfg, avg_bits, n_tokens=2048, budget_s=8.0):
    """The oracle planner (16 streams of the layer from their 4096-vector calibration sets) and
    the oracle encode (project, scale, quantize, pack) of n_tokens per stream, on one host thread."""
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")
    r = subprocess.run([sys.executable, "-c", _ORACLE_ENCODE_CHILD, ROOT, cfg.name, str(avg_bits), str(n_tokens),
                        str(budget_s)], capture_output=True, text=True, env=env, timeout=600)
    if r.returncode != 0:
        return {"error": r.stderr[-300:]}
    d = json.loads(r.stdout.strip().splitlines()[-1])
    toks = d["reps"] * n_tokens
    return {"encode_mtok_s": round(toks / d["encode_seconds"] / 1e6, 6),
            "encode_input_gbs": round(toks * cfg.n_kv_heads * 2 * 128 * 2 / d["encode_seconds"] / 1e9, 6),
            "planner_seconds_per_layer": round(d["plan_seconds"], 3), "cores": 1,
            "sample": f"oracle encode of {n_tokens} tokens x {cfg.n_kv_heads} kv-heads x K|V (numpy fp64, 1 thread), "
                      f"{d['reps']} repetitions in {d['encode_seconds']:.1f} s; oracle planner of the layer's "
                      f"{2 * cfg.n_kv_heads} streams from 4096 calibration vectors each"}


def oracle_code_agreement(p, cache, kd, vd, cfg, n_words, n_tokens=4096):
    """The oracle encode of the first n_tokens of every stream with the library's plan (basis,
    widths, scales), against the codes the GPU wrote into `cache`: codes equal, codes one level
    off at a decision threshold (|h/Delta - (k + 1/2)| <= 1e-4 relative), and any other
    difference (must be none)."""
    from oracle import aatc_oracle as O
    import torch
    torch.cuda.synchronize()
    host = cache.cpu().numpy().view(np.uint32)
    B, Tc = kd.shape[0], kd.shape[1]
    n = min(n_tokens, Tc)
    tot = mis = far = 0
    for h in range(cfg.n_kv_heads):
        for kind, x in ((0, kd), (1, vd)):
            bits = p["bits"][0, h, kind].astype(np.int64)
            ub = W.to_bf16(p["basis"][0, h, kind]).astype(np.float64)
            xs = x[0, :n, h].float().cpu().numpy().astype(np.float64)
            codes, _, t = O.encode_stream(xs, ub, bits, p["scales"][0, h, kind].astype(np.float64))
            rec, _ = O.cache_records(host, B, cfg.n_kv_heads, Tc, n_words, 0, h, kind, 0, n)
            got = O.unpack_records(rec, bits)
            keep = bits > 0
            diff = got[:, keep] - codes[:, keep]
            tk = t[:, keep]
            thr = np.floor(tk) + 0.5
            near = np.abs(tk - thr) <= 1e-4 * np.abs(thr)
            tot += int(keep.sum()) * n
            mis += int(np.count_nonzero(diff))
            far += int(np.count_nonzero((diff != 0) & ~((np.abs(diff) == 1) & near)))
    return {"codes": tot, "near_threshold_one_level": mis - far, "other_differences": far,
            "fraction": mis / max(tot, 1),
            "sample": f"first {n} tokens of sequence 0, all {cfg.n_kv_heads} kv-heads x K|V, library plan"}


def cpu_baseline(cfg, avg_bits, budget_s=15.0, n_tokens=4096, all_cores_s=0.0):
    """Oracle decode (unpack + fp32 dequant + fp64 attention) timed on one host thread over a
    bounded sample: all 32 q-heads over the first n_tokens tokens, repeated for ~budget_s s.
    With all_cores_s > 0, also one single-threaded oracle process per host core at once for
    ~all_cores_s s (aggregate rate, reported under "all_cores")."""
    sample = oracle_sample(cfg, avg_bits, n_tokens)
    what = f"oracle decode of all {cfg.n_q_heads} q-heads over the first {n_tokens} tokens (numpy fp64"
    with tempfile.TemporaryDirectory() as td:
        path = os.path.join(td, "sample.npz")
        np.savez(path, **sample)
        res, err = _run_oracle_children(path, budget_s, 1)
        if err is not None or res["seconds"] <= 0:
            return {"value": None, "unit": "GB/s", "cores": 1, "kind": "oracle", "error": err}
        line = {"value": round(res["bytes"] / res["seconds"] / 1e9, 6), "unit": "GB/s", "cores": 1, "kind": "oracle",
                "sample": f"{what}, 1 thread), {res['decodes']} repetitions in {res['seconds']:.1f} s"}
        if all_cores_s > 0:
            n_proc = len(os.sched_getaffinity(0))
            allc, err = _run_oracle_children(path, all_cores_s, n_proc)
            if err is None and allc["seconds"] > 0:
                line["all_cores"] = {"value": round(allc["bytes"] / allc["seconds"] / 1e9, 6), "unit": "GB/s",
                                     "cores": n_proc,
                                     "sample": f"{what}, {n_proc} single-threaded processes at once), "
                                               f"{allc['decodes']} repetitions in {allc['seconds']:.1f} s"}
    return line


def run_reference(args):
    ws_, rank = _dist()
    if rank != 0:
        return
    cfg = W.CONFIGS[args.config]
    avg_bits = cfg.avg_bits[-1] if args.bits is None else args.bits
    per_step = max(1.0, min(10.0, 120.0 / max(1, args.steps + args.warmup)))
    times = []
    walls = []
    res = None
    for s in range(args.warmup + args.steps):
        t0 = time.perf_counter()
        res = cpu_baseline(cfg, avg_bits, budget_s=per_step, n_tokens=2048)
        if s >= args.warmup:
            times.append(res)
            walls.append(time.perf_counter() - t0)
    vals = [r["value"] for r in times if r.get("value")]
    value = float(np.mean(vals)) if vals else None
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": ws_, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(float(np.mean(walls)) * 1e3, 1) if walls else None,
        "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": cfg.workload, "avg_bits": avg_bits, "batch": cfg.batch, "n_ctx": cfg.n_ctx},
        "cpu_baseline": {"value": value, "unit": "GB/s", "cores": 1, "kind": "oracle",
                         "sample": (res or {}).get("sample", "")},
        "e2e": {"value": value, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_profile_once(args):
    """Minimal launch sequence for ncu captures: one encode, two decodes, one bf16 decode (with
    --config llama_stack: one 131072-token layer of the stack)."""
    import torch
    import paper_2608_14191_gb300 as aatc
    from paper_2608_14191_gb300 import build as bld
    bld.build()
    aatc.load()
    dev = torch.device("cuda", 0)
    cfg = W.CONFIGS[args.config]
    if cfg.n_layers > 1:
        import dataclasses
        cfg = dataclasses.replace(cfg, n_layers=1)
    avg_bits = cfg.avg_bits[-1] if args.bits is None else args.bits
    B, T = cfg.batch, cfg.n_ctx
    plan, _ = build_case(aatc, cfg, avg_bits, dev)
    kd, vd = W.kv_device(cfg, 0, B, T, dev)
    qs = W.queries_device(cfg, 0, B, 2, dev)
    cache = plan.new_cache(B, T, dev)
    aatc.encode(plan, 0, kd, vd, cache, 0, T)
    for i in range(2):
        aatc.decode_attention(plan, 0, qs[i], cache, T, T)
    aatc.bf16_decode_attention(kd, vd, qs[0], T)
    torch.cuda.synchronize()
    assert plan.device_error() == 0
    print(json.dumps({"profile_once": cfg.name, "decode_bytes": decode_bytes(plan, cfg, B, T)}))


def run_profile_groups():
    """Minimal launch sequence of the head-group path for ncu captures: the Llama-shaped layer
    with two groups of four kv-heads, one encode and two decodes."""
    import torch
    import paper_2608_14191_gb300 as aatc
    from paper_2608_14191_gb300 import build as bld
    bld.build()
    aatc.load()
    dev = torch.device("cuda", 0)
    cfg = W.CONFIGS["llama_layer"]
    plan, _ = group_plan_for(aatc, cfg, 4)
    T = cfg.n_ctx
    kd, vd = W.kv_device(cfg, 0, 1, T, dev)
    qs = W.queries_device(cfg, 0, 1, 2, dev)
    cache = plan.new_cache(1, T, dev)
    aatc.encode(plan, 0, kd, vd, cache, 0, T)
    for i in range(2):
        aatc.decode_attention(plan, 0, qs[i], cache, T, T)
    torch.cuda.synchronize()
    assert plan.device_error() == 0
    print(json.dumps({"profile_groups": "llama layer, 2 groups x 4 kv-heads, 32768 tokens"}))


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", default="llama_layer", choices=sorted(W.CONFIGS))
    ap.add_argument("--bits", type=float, default=None)
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--profile-once", action="store_true", help="one encode + two decodes, for ncu")
    ap.add_argument("--profile-hidden", action="store_true", help="one encode from hidden states, for ncu")
    ap.add_argument("--profile-prefill", action="store_true", help="one Qwen-shaped prefill at batch 2, for ncu")
    ap.add_argument("--profile-groups", action="store_true", help="one head-group encode + two decodes, for ncu")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.profile_once:
        run_profile_once(args)
    elif args.profile_hidden:
        import torch
        import paper_2608_14191_gb300 as aatc
        from paper_2608_14191_gb300 import build as bld
        bld.build()
        aatc.load()
        hidden_encode_timing(aatc, torch.device("cuda", 0), iters=0, warmup=1)
        print(json.dumps({"profile_hidden": "llama layer input, d_model 4096, 32768 tokens"}))
    elif args.profile_groups:
        run_profile_groups()
    elif args.profile_prefill:
        import torch
        import paper_2608_14191_gb300 as aatc
        from paper_2608_14191_gb300 import build as bld
        bld.build()
        aatc.load()
        prefill_timing(aatc, torch.device("cuda", 0), iters=0, batch=2)
        print(json.dumps({"profile_prefill": "qwen layer, batch 2 x 8192, causal"}))
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
