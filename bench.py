#!/usr/bin/env python
"""Throughput benchmark of the TransX serving hot path on GB300.

One step = one pass of the whole path over one synthetic serving batch:
refresh the behavior K/V cache of every request in place (projection of all
rows + attention-pooled anchor), append new behavior rows, score every
candidate through the decoder stack and the action head, and rank each
request's candidates.  `value` is candidates per second over the K timed steps
(inputs resident in HBM); `e2e` is the same through the public API with host
buffers (pinned host -> device copies of the step's inputs and the device ->
host read of probabilities and rankings inside the timed region).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl txs|reference]

Under torchrun every rank runs its own batch (requests shard across GPUs with
no collective on the data path); rank 0 prints one JSON line.
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
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2607_28940_gb300 import workload as W  # noqa: E402

METRIC = "candidates scored/sec per GB300 and p50 request latency vs behavior length L"
# the largest configuration that fits one GPU: 64 requests, 4 layers, d = 512,
# L_r ~ U[1024, 16384], M = 1000 packed varlen
HEADLINE = "ragged_bf16"
DW_WORKLOAD = "small_bf16"             # model of the Deep & Wide head measurement
LAT_WORKLOAD = "ragged_bf16"          # the long-history model for the latency-vs-L sweep
LAT_LENGTHS = (1024, 2048, 4096, 8192, 16384)
LAT_M = 1000
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0}

# DRAM traffic per launch measured with ncu (dram__bytes_read.sum +
# dram__bytes_write.sum) for the kernel classes that can be dominant, with the
# sha256 prefix of the kernel source at capture time; a source change voids it.
# (workload, mode, class) -> (bytes per launch, source sha256[:12]), each from
# one --set full capture of that class's kernel on that workload.
NCU_TRAFFIC = {
    # rebuild of the 262,144 rows of mid_bf16 (272.7 MB read + 2.092 GB written)
    # scaled by rows to the 525,811 of ragged_bf16, plus the 512-row append
    # (4.8 MB + 0.04 MB), averaged over the two launches of a step
    ("ragged_bf16", "local_global", "gemm_kv_build"): (2.374e+09, "d7e79a9337e8"),
    ("mid_bf16", "full", "attn_cross"): (873.9e6, "db3c1a34b26e"),
    ("sweep_bf16", "full", "attn_cross"): (317.1e6, "db3c1a34b26e"),
}


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=300)
    p.add_argument("--warmup", type=int, default=20)
    p.add_argument("--impl", default="txs", choices=["txs", "reference"])
    p.add_argument("--workload", default=HEADLINE, choices=sorted(W.WORKLOADS))
    p.add_argument("--mode", default="local_global", choices=["local_global", "full"])
    p.add_argument("--no-extras", action="store_true", help="skip latency sweep, e2e and CPU baseline")
    p.add_argument("--section", choices=["encoder", "deep_wide", "events", "sweep", "latency"],
                   help="run only this extra section (one JSON object) and exit")
    p.add_argument("--enc-len", type=int, default=0,
                   help="tokens per user of the encoder section (default: the workload's)")
    return p.parse_args()


def describe(wl: W.Workload, mode: str) -> str:
    return (f"{wl.name}: R={wl.n_req} requests, {wl.n_layers} layers, d={wl.d_model}, {wl.n_heads} heads, "
            f"FFN {wl.d_ff}, L={wl.L}, M={wl.M}, +{wl.dL} appended rows/request, S={wl.n_ctx}, k={wl.n_actions}, "
            f"L_local={wl.l_local}, {mode.upper()} cross-attention")


def step_config(wl: W.Workload, mode: str, world: int) -> dict:
    """The `config` object of the JSON line; both arms print the same one."""
    L, M, dL = W.sizes(wl)
    es = 2 if wl.dtype == "bf16" else 4
    cache_rows = int((L + wl.capacity_extra).sum())
    big = es * wl.d_model * (int(L.sum() + dL.sum() + M.sum()) + 2 * wl.n_layers * cache_rows) > (129 << 20)
    return {"workload": describe(wl, mode), "global_batch": int(M.sum()) * world,
            "requests_per_gpu": wl.n_req, "seq_len": int(L.max()),
            "step": "in-place cache rebuild + append (one call, side stream) + score + rank; the part "
                    "of scoring that does not read the cache overlaps the refresh",
            "l2": "flushed before every timed step (256 MiB device write, untimed)" +
                  ("; the step's inputs and cache exceed L2 as well" if big else ""),
            "parallelism": f"request-sharded replicas x{world} (no data-path collective)"}


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return {"hbm_gbs": float(p["hbm_gbs"]), "bf16_tflops": float(p["bf16_tflops"]),
                "bf16_tflops_sustained": float(p.get("bf16_tflops_sustained", p["bf16_tflops"]))}, "measured"
    except Exception:
        return dict(FALLBACK_PEAKS, bf16_tflops_sustained=1700.0), "fallback"


# ---------------------------------------------------------------- algorithmic work per class

def algorithmic(wl: W.Workload, mode: int, L: np.ndarray, M: np.ndarray, dL: np.ndarray, fused_lg: bool = False):
    """Per-step algorithmic (flops, bytes) of each kernel class: what the method
    must compute and move (bf16 operands, fp32 vectors), independent of how the
    kernels tile it.  fused_lg: the LOCAL_GLOBAL attention of the candidate
    rows runs inside the query projection (class gemm_q_attn_lg) and only the
    context-token rows go through a separate attention launch (attn_cross)."""
    es = 2 if wl.dtype == "bf16" else 4
    d, F, nL, H, S, k = wl.d_model, wl.d_ff, wl.n_layers, wl.n_heads, wl.n_ctx, wl.n_actions
    R = wl.n_req
    n_cand = int(M.sum())
    N = n_cand + R * S
    sumL, sumdL = int(L.sum()), int(dL.sum())

    def gemm(m, n, kk, res=False, out_es=es):
        flops = 2.0 * m * n * kk
        byt = es * (m * kk + n * kk) + out_es * m * n + (es * m * n if res else 0) + 4 * n
        return flops, byt

    out = {}

    def add(name, fb):
        f0, b0 = out.get(name, (0.0, 0.0))
        out[name] = (f0 + fb[0], b0 + fb[1])

    for rows in (sumL, sumdL):   # rebuild, append
        add("gemm_kv_build", gemm(rows, 2 * nL * d, d))
        add("pool", (4.0 * rows * d, es * rows * d + 4 * R * (d + 2)))
        add("global_kv", (2.0 * R * 2 * nL * d * d, es * 2 * nL * d * d + 4 * R * d * (1 + 2 * nL)))
    add("pack", (2.0 * n_cand * d * k, es * 2 * N * d + 4 * n_cand * k))
    L_after = L + dL
    W_keys = np.minimum(L_after, wl.l_local) + 1 if mode == 0 else L_after
    rows_per_req = M + S
    for l in range(nL):
        add("gemm_qkv", gemm(N, 3 * d, d))
        add("attn_serving", (4.0 * d * (n_cand * (S + 1) + R * S * S), es * (N * 3 * d + N * d)))
        add("gemm_oproj_ln", gemm(N, d, d, res=True))
        kv_bytes = float((W_keys * 2 * d * es).sum())
        if fused_lg:
            # query projection and the candidate rows' attention in one kernel
            # (the query of a candidate row never goes to memory); the context
            # rows' queries go out and their attention runs separately
            qf, qb = gemm(N, d, d)
            add("gemm_q_attn_lg", (qf + float((4.0 * d * M * W_keys).sum()), qb + kv_bytes))
            add("attn_cross", (float((4.0 * d * S * W_keys).sum()), es * 3 * R * S * d + kv_bytes))
        else:
            add("gemm_q", gemm(N, d, d))
            add("attn_cross", (float((4.0 * d * rows_per_req * W_keys).sum()), es * 2 * N * d + kv_bytes))
        add("gemm_oproj_ln", gemm(N, d, d, res=True))
        add("gemm_ffn1_gelu", gemm(N, F, d))
        add("gemm_ffn2_ln", gemm(N, d, F, res=True))
    add("rank", (float((M.astype(np.float64) ** 2).sum()), 4.0 * n_cand * (k + 1)))
    return out


# ---------------------------------------------------------------- clocks

CLOCK_FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
                "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
                "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")


class ClockSampler:
    """nvidia-smi sampling in the background while the GPU works."""

    def __init__(self, index: int):
        self.path = tempfile.mktemp(suffix=".csv")
        self.proc = None
        self.index = index

    def start(self):
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={CLOCK_FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        self.t0 = time.time()

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.f.close()

    def summary(self):
        rows = []
        try:
            with open(self.path) as f:
                for line in f:
                    parts = [p.strip() for p in line.split(",")]
                    if len(parts) >= 10:
                        rows.append(parts)
        except Exception:
            pass
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        sm = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        mx = [float(r[3]) for r in rows if r[3].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[6 + i].lower() == "active"})
        pw = [float(r[4]) for r in rows if r[4].replace(".", "").isdigit()]
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows), "power_w_max": max(pw) if pw else None}


# ---------------------------------------------------------------- the GPU arm

def run_txs(args, rank, world):
    import torch
    from paper_2607_28940_gb300 import build as B
    from paper_2607_28940_gb300 import txs

    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if not os.path.exists(txs.LIB_PATH):
        B.build()
    mode = txs.LOCAL_GLOBAL if args.mode == "local_global" else txs.FULL
    from paper_2607_28940_gb300 import shard
    wl = W.WORKLOADS[args.workload]                          # per-rank batch shape
    # the job is world * R requests; each rank takes its own contiguous block
    b = W.batch(shard.global_workload(wl, world), requests=shard.shard_requests(wl.n_req, rank, world))
    weights = W.weights(wl)                                  # one model, replicated
    dt = txs.torch_dtype(wl.dtype)
    n_cand = int(b.cand_off[-1])
    full_off = b.beh_off

    model = txs.Model(wl, weights, mode)
    beh = txs.to_device(b.beh, dt)
    app = txs.to_device(b.app, dt)
    cand = txs.to_device(b.cand, dt)
    ctx = txs.to_device(b.ctx.reshape(-1, wl.d_model), dt) if wl.n_ctx else None
    cache = txs.KVCache(model, full_off, beh, capacity_extra=wl.capacity_extra)
    ws = torch.empty(txs.workspace_bytes(model, wl.n_req, n_cand), dtype=torch.uint8, device="cuda")
    logits = torch.empty((n_cand, wl.n_actions), dtype=torch.float32, device="cuda")
    probs = torch.empty_like(logits)
    ranks = torch.empty(n_cand, dtype=torch.int32, device="cuda")
    flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
    stream = torch.cuda.current_stream()

    def step(start_ev=None, beh_t=beh, app_t=app, cand_t=cand, ctx_t=ctx):
        cache.rebuild_append(full_off, beh_t, b.app_off, app_t)
        txs.score(model, cache, b.cand_off, cand_t, ctx_t, workspace=ws, out_logits=logits, out_probs=probs)
        txs.rank(b.cand_off, probs, wl.n_actions, 0, 0, out=ranks)

    # The timed step: the same calls, with the cache refresh on a side stream
    # (after the step's start event, i.e. after the previous step's reads of
    # the cache) overlapping the part of scoring that does not read the cache
    # (txs_score_candidates_after waits for it before the first
    # cross-attention).
    side = torch.cuda.Stream()
    ready = torch.cuda.Event()

    def step_overlap(start_ev):
        side.wait_event(start_ev)
        with torch.cuda.stream(side):
            cache.rebuild_append(full_off, beh, b.app_off, app)
            ready.record(side)
        txs.score(model, cache, b.cand_off, cand, ctx, workspace=ws, out_logits=logits, out_probs=probs,
                  cache_ready=ready)
        txs.rank(b.cand_off, probs, wl.n_actions, 0, 0, out=ranks)

    def barrier():
        torch.cuda.synchronize()
        if world > 1:
            torch.distributed.barrier()

    def timed(fn, steps, do_flush=True):
        evs = []
        for _ in range(steps):
            if do_flush:
                flush.zero_()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            fn(e0)
            e1.record(stream)
            evs.append((e0, e1))
        torch.cuda.synchronize()
        return [a.elapsed_time(c) for a, c in evs]

    clocks = ClockSampler(local)
    clocks.start()
    for _ in range(max(args.warmup, 3)):
        e = torch.cuda.Event()
        e.record(stream)
        step_overlap(e)
    barrier()
    wall0 = time.perf_counter()
    ms = timed(step_overlap, args.steps)
    barrier()
    wall = time.perf_counter() - wall0
    clocks.stop()
    st = model.device_status()
    if st != txs.TXS_OK:
        raise RuntimeError(f"device status {st} after timed region")

    total_ms_max = shard.reduce_max(float(sum(ms)), device="cuda")
    value = world * n_cand * args.steps / (total_ms_max / 1e3)

    # per-kernel breakdown: the same K steps again, on one stream, with event
    # pairs around every launch
    txs.profile_enable(True)
    timed(step, args.steps)
    prof = txs.profile_collect()
    txs.profile_enable(False)
    launches_per_step = sum(c for _, c in prof.values()) / args.steps

    out = {"metric": METRIC, "value": value, "unit": "candidates/s", "n_gpus": world, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": total_ms_max / args.steps, "higher_is_better": True,
           "scaling": "weak", "vs_baseline": None, "dtype": "bf16" if wl.dtype == "bf16" else "f32",
           "data": "synthetic (seeded N(0,1) inputs, N(0,0.02) weights; shapes of the paper's serving setting)"}
    out["config"] = step_config(wl, args.mode, world)
    out["wall_s_timed_region"] = wall
    out["gpu_launches"] = int(round(launches_per_step * args.steps))
    out["clocks"] = clocks.summary()

    peaks, peak_src = load_peaks()
    alg = algorithmic(wl, mode, b.L, b.M, b.dL, fused_lg="gemm_q_attn_lg" in prof)
    kern = {}
    for name, (tot, cnt) in prof.items():
        per_step_ms = tot / args.steps
        f, by = alg.get(name, (0.0, 0.0))
        t_s = per_step_ms / 1e3
        kern[name] = {"ms_per_step": per_step_ms, "launches_per_step": cnt / args.steps,
                      "share": tot / max(sum(v[0] for v in prof.values()), 1e-12),
                      "tflops": f / t_s / 1e12 if t_s > 0 else None, "gbs": by / t_s / 1e9 if t_s > 0 else None}
    out["kernels"] = kern
    dom = max(prof.items(), key=lambda kv: kv[1][0])[0]
    f, by = alg[dom]
    per_launch_ms = prof[dom][0] / prof[dom][1]
    launches = prof[dom][1] / args.steps
    t_tensor = f / (peaks["bf16_tflops"] * 1e12)
    t_hbm = by / (peaks["hbm_gbs"] * 1e9)
    if t_tensor >= t_hbm:
        achieved = f / launches / (per_launch_ms / 1e3) / 1e12
        roof = {"bound": "tensor", "achieved": achieved, "peak": peaks["bf16_tflops"], "unit": "TFLOP/s"}
    else:
        achieved = by / launches / (per_launch_ms / 1e3) / 1e9
        roof = {"bound": "hbm", "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s"}
    roof["frac"] = roof["achieved"] / roof["peak"]
    tr = NCU_TRAFFIC.get((args.workload, args.mode, dom))
    src_file = ("k_gemm_ln.cu" if dom in ("gemm_oproj_ln", "gemm_ffn2_ln") and wl.dtype == "bf16" and
                wl.d_model in (256, 512) else
                "k_gemm_tc.cu" if dom.startswith("gemm") else
                "k_attn_tc.cu" if (dom == "attn_cross" and args.mode == "full" and wl.dtype == "bf16") else
                "k_score.cu" if dom in ("pack", "rank") else
                "k_cache.cu" if dom in ("pool", "global_kv") else "k_attn.cu")
    src_sha = hashlib.sha256(open(os.path.join(ROOT, "paper_2607_28940_gb300", "csrc", src_file),
                                  "rb").read()).hexdigest()[:12]
    roof["traffic"] = tr[0] if tr and tr[1] == src_sha else None
    roof["kernel"] = dom
    roof["peak_source"] = f"{peak_src} ({'burst' if roof['bound'] == 'tensor' else 'copy'})"
    roof["algorithmic_per_launch"] = {"flops": f / launches, "bytes": by / launches}
    out["roofline"] = roof

    if not args.no_extras:
        out["score_only"] = score_only(txs, torch, model, cache, b, cand, ctx, ws, logits, probs, ranks, wl,
                                       timed, args.steps)
        out["e2e"] = e2e(txs, torch, model, cache, b, wl, args, dt, logits, probs, ranks, ws, world)
        if rank == 0:
            out["latency_vs_L"] = latency_sweep(txs, torch)
            out["events"] = events_bench(txs, torch)
            out["encoder"] = encoder_bench(txs, torch, peaks, peak_src)
            out["deep_wide"] = deep_wide_bench(txs, torch)
            out["sweep"] = sweep_bench(txs, torch, peaks, peak_src)
            out["cpu_baseline"] = cpu_baseline(args.workload, budget_s=15.0)
    return out


def score_only(txs, torch, model, cache, b, cand, ctx, ws, logits, probs, ranks, wl, timed, steps):
    def fn(_start=None):
        txs.score(model, cache, b.cand_off, cand, ctx, workspace=ws, out_logits=logits, out_probs=probs)
        txs.rank(b.cand_off, probs, wl.n_actions, 0, 0, out=ranks)
    ms = timed(fn, steps)
    n = int(b.cand_off[-1])
    return {"value": n * steps / (sum(ms) / 1e3), "unit": "candidates/s", "ms_per_call": sum(ms) / steps,
            "what": "score + rank against the prebuilt cache (the online part of the path), L2 flushed"}


def e2e(txs, torch, model, cache, b, wl, args, dt, logits, probs, ranks, ws, world):
    """The step through the public API from pinned host buffers, reading results back."""
    pin = lambda a: torch.from_numpy(np.ascontiguousarray(a, np.float32)).to(dt).pin_memory()
    h_beh, h_app, h_cand = pin(b.beh), pin(b.app), pin(b.cand)
    h_ctx = pin(b.ctx.reshape(-1, wl.d_model)) if wl.n_ctx else None
    d_beh = torch.empty(h_beh.shape, dtype=dt, device="cuda")
    d_app = torch.empty(h_app.shape, dtype=dt, device="cuda")
    d_cand = torch.empty(h_cand.shape, dtype=dt, device="cuda")
    d_ctx = torch.empty(h_ctx.shape, dtype=dt, device="cuda") if h_ctx is not None else None
    h_probs = torch.empty(probs.shape, dtype=torch.float32).pin_memory()
    h_ranks = torch.empty(ranks.shape, dtype=torch.int32).pin_memory()
    n = int(b.cand_off[-1])

    main = torch.cuda.current_stream()
    side = torch.cuda.Stream()
    ready = torch.cuda.Event()

    def one():
        # behavior rows in and the cache refresh on a side stream, candidates
        # in and the cache-independent start of scoring on the main stream
        side.wait_stream(main)
        with torch.cuda.stream(side):
            d_beh.copy_(h_beh, non_blocking=True)
            d_app.copy_(h_app, non_blocking=True)
            cache.rebuild_append(b.beh_off, d_beh, b.app_off, d_app)
            ready.record(side)
        d_cand.copy_(h_cand, non_blocking=True)
        if d_ctx is not None:
            d_ctx.copy_(h_ctx, non_blocking=True)
        txs.score(model, cache, b.cand_off, d_cand, d_ctx, workspace=ws, out_logits=logits, out_probs=probs,
                  cache_ready=ready)
        txs.rank(b.cand_off, probs, wl.n_actions, 0, 0, out=ranks)
        h_probs.copy_(probs, non_blocking=True)
        h_ranks.copy_(ranks, non_blocking=True)
        main.synchronize()

    for _ in range(3):
        one()
    steps = max(args.steps // 2, 10)
    t0 = time.perf_counter()
    for _ in range(steps):
        one()
    from paper_2607_28940_gb300 import shard
    dt_s = shard.reduce_max(time.perf_counter() - t0, device="cuda")
    h2d = sum(x.numel() * x.element_size() for x in (h_beh, h_app, h_cand) + ((h_ctx,) if h_ctx is not None else ()))
    d2h = h_probs.numel() * 4 + h_ranks.numel() * 4
    return {"value": world * n * steps / dt_s, "unit": "candidates/s", "h2d_bytes_per_step": int(h2d),
            "d2h_bytes_per_step": int(d2h), "steps": steps,
            "what": "pinned host -> device inputs, full step (cache refresh and its inputs on a side stream), "
                    "device -> host probs and ranks, synchronised per step"}


def latency_sweep(txs, torch):
    """p50 latency of one request (score + rank of M candidates) against prebuilt
    caches of growing behavior length L, both key-set modes."""
    base = W.WORKLOADS[LAT_WORKLOAD]
    weights = W.weights(base)
    res = {"model": f"{LAT_WORKLOAD} layers/width (d={base.d_model}, {base.n_layers} layers), R=1, M={LAT_M}",
           "unit": "ms", "note": "CUDA events, weights L2-warm as in steady serving; *_graph_replay: the same "
                                 "score + rank captured into a CUDA graph once per length and replayed"}
    side = torch.cuda.Stream()
    for mode_name, mode in (("local_global", txs.LOCAL_GLOBAL), ("full", txs.FULL)):
        model = txs.Model(base, weights, mode)
        p50, p50_graph = {}, {}
        for L in LAT_LENGTHS:
            wl = W.with_sizes(base, n_req=1, L=L, M=LAT_M, dL=0)
            b = W.batch(wl)
            dt = txs.torch_dtype(wl.dtype)
            cache = txs.KVCache(model, b.beh_off, txs.to_device(b.beh, dt))
            cand = txs.to_device(b.cand, dt)
            ctx = txs.to_device(b.ctx.reshape(-1, wl.d_model), dt)
            ws = torch.empty(txs.workspace_bytes(model, 1, LAT_M), dtype=torch.uint8, device="cuda")
            lg = torch.empty((LAT_M, wl.n_actions), dtype=torch.float32, device="cuda")
            pr = torch.empty_like(lg)
            rk = torch.empty(LAT_M, dtype=torch.int32, device="cuda")
            def call():
                txs.score(model, cache, b.cand_off, cand, ctx, workspace=ws, out_logits=lg, out_probs=pr)
                txs.rank(b.cand_off, pr, wl.n_actions, 0, 0, out=rk)

            def p50_of(fn):
                times = []
                with torch.cuda.stream(side):
                    for i in range(40):
                        e0 = torch.cuda.Event(enable_timing=True)
                        e1 = torch.cuda.Event(enable_timing=True)
                        e0.record()
                        fn()
                        e1.record()
                        e1.synchronize()
                        if i >= 10:
                            times.append(e0.elapsed_time(e1))
                return statistics.median(times)
            p50[str(L)] = p50_of(call)
            # the same call captured once into a CUDA graph and replayed (a
            # server keeps one graph per slate shape)
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=side):
                call()
            p50_graph[str(L)] = p50_of(g.replay)
            del g
            cache.close()
        res[mode_name] = p50
        res[f"{mode_name}_graph_replay"] = p50_graph
        res[f"{mode_name}_ratio_16384_over_1024"] = p50["16384"] / p50["1024"]
        model.close()
    return res


EV_WORKLOAD = "mid_bf16"     # model dims of the streaming multi-event measurement
EV_L, EV_T, EV_M = 8192, 64, 256


def events_bench(txs, torch):
    """Streaming multi-event scoring (txs_score_events): one user's stream of
    EV_L rows cached once, EV_T events at sorted prefix ends, EV_M candidates
    each; candidates/s and events/s over repeated calls, L2 flushed before
    each call, plus the per-class time of one call."""
    base = W.WORKLOADS[EV_WORKLOAD]
    wl = W.with_sizes(base, n_req=1, L=EV_L, M=1, dL=0)
    res = {"workload": f"{EV_WORKLOAD} model (d={base.d_model}, {base.n_layers} layers), one user with L={EV_L} "
                       f"rows, T={EV_T} events at uniform sorted prefix ends, {EV_M} candidates per event",
           "unit": "candidates/s"}
    ev = W.events(wl, EV_L, EV_T, EV_M, 20267)
    dt = txs.torch_dtype(wl.dtype)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
    for mode_name, mode in (("local_global", txs.LOCAL_GLOBAL), ("full", txs.FULL)):
        model = txs.Model(wl, W.weights(wl), mode)
        beh = txs.to_device(ev.beh, dt)
        cache = txs.KVCache(model, np.array([0, EV_L], dtype=np.int32), beh)
        cand = txs.to_device(ev.cand, dt)
        ctx = txs.to_device(ev.ctx.reshape(-1, wl.d_model), dt)
        n_cand = int(ev.cand_off[-1])
        ws = torch.empty(txs.events_workspace_bytes(model, EV_T, n_cand, int(ev.ends.max())), dtype=torch.uint8,
                         device="cuda")
        lg = torch.empty((n_cand, wl.n_actions), dtype=torch.float32, device="cuda")
        pr = torch.empty_like(lg)
        call = lambda: txs.score_events(model, cache, 0, beh, ev.ends, ev.cand_off, cand, ctx, workspace=ws,
                                        out_logits=lg, out_probs=pr)
        for _ in range(3):
            call()
        times = []
        for _ in range(10):
            flush.zero_()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record()
            call()
            e1.record()
            e1.synchronize()
            times.append(e0.elapsed_time(e1))
        txs.profile_enable(True)
        call()
        torch.cuda.synchronize()
        prof = txs.profile_collect()
        txs.profile_enable(False)
        ms = statistics.median(times)
        res[mode_name] = {"ms_per_call": ms, "candidates_per_s": n_cand / (ms / 1e3),
                          "events_per_s": EV_T / (ms / 1e3),
                          "kernels_ms": {k: v[0] for k, v in prof.items()}}
        if model.device_status() != txs.TXS_OK:
            raise RuntimeError("device status after the events measurement")
        cache.close()
        model.close()
    return res


SWEEP_WORKLOAD = "sweep_bf16"   # R = 16 requests x 8192 behavior rows, d = 512, 4 layers
SWEEP_M = (64, 256, 1024, 4096)
SWEEP_DL = (1, 2, 4, 8, 16, 32, 64)


def sweep_bench(txs, torch, peaks, peak_src):
    """The sweep configuration: score + rank latency and candidates/s for
    M in SWEEP_M candidates per request against one prebuilt cache (both
    key-set modes; FULL with the roofline of its cross-attention), and the
    incremental append of dL in SWEEP_DL rows per request against a full
    rebuild of the cache (App. D: an append scales with the new rows)."""
    base = W.WORKLOADS[SWEEP_WORKLOAD]
    weights = W.weights(base)
    dt = txs.torch_dtype(base.dtype)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
    b0 = W.batch(base, M_override=SWEEP_M[0])
    beh = txs.to_device(b0.beh, dt)
    L = int(b0.L[0])
    d, nL = base.d_model, base.n_layers
    res = {"workload": f"{SWEEP_WORKLOAD}: R={base.n_req} requests x L={L} rows, d={d}, {nL} layers; "
                       f"M per request in {list(SWEEP_M)}; appends of dL rows per request in {list(SWEEP_DL)}",
           "unit": "ms"}

    def timed(fn, reps, flush_l2=True):
        for _ in range(3):
            fn()
        times = []
        for _ in range(reps):
            if flush_l2:
                flush.zero_()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record()
            fn()
            e1.record()
            e1.synchronize()
            times.append(e0.elapsed_time(e1))
        return statistics.median(times)

    for mode_name, mode in (("local_global", txs.LOCAL_GLOBAL), ("full", txs.FULL)):
        model = txs.Model(base, weights, mode)
        cache = txs.KVCache(model, b0.beh_off, beh)
        rows = {}
        for M in SWEEP_M:
            b = W.batch(base, M_override=M)
            cand = txs.to_device(b.cand, dt)
            ctx = txs.to_device(b.ctx.reshape(-1, d), dt)
            n = int(b.cand_off[-1])
            ws = torch.empty(txs.workspace_bytes(model, base.n_req, n), dtype=torch.uint8, device="cuda")
            lg = torch.empty((n, base.n_actions), dtype=torch.float32, device="cuda")
            pr = torch.empty_like(lg)
            rk = torch.empty(n, dtype=torch.int32, device="cuda")

            def call():
                txs.score(model, cache, b.cand_off, cand, ctx, workspace=ws, out_logits=lg, out_probs=pr)
                txs.rank(b.cand_off, pr, base.n_actions, 0, 0, out=rk)
            ms = timed(call, 10)
            row = {"ms_per_call": ms, "candidates_per_s": n / (ms / 1e3)}
            if mode == txs.FULL:
                txs.profile_enable(True)
                call()
                torch.cuda.synchronize()
                prof = txs.profile_collect()
                txs.profile_enable(False)
                a_ms = prof.get("attn_cross", (0.0, 0))[0]
                fl = 4.0 * n * L * d * nL          # candidate rows only
                by = 2.0 * nL * (2 * base.n_req * L * d + 2 * n * d)
                t_t, t_h = fl / (peaks["bf16_tflops"] * 1e12), by / (peaks["hbm_gbs"] * 1e9)
                if t_t >= t_h:
                    ach = fl / (a_ms / 1e3) / 1e12
                    row["roofline_attn_cross"] = {"bound": "tensor", "achieved": ach, "peak": peaks["bf16_tflops"],
                                                  "unit": "TFLOP/s", "frac": ach / peaks["bf16_tflops"]}
                else:
                    ach = by / (a_ms / 1e3) / 1e9
                    row["roofline_attn_cross"] = {"bound": "hbm", "achieved": ach, "peak": peaks["hbm_gbs"],
                                                  "unit": "GB/s", "frac": ach / peaks["hbm_gbs"]}
                row["roofline_attn_cross"].update({"kernel": "attn_cross", "ms": a_ms,
                                                   "peak_source": f"{peak_src} ({'burst' if t_t >= t_h else 'copy'})"})
            rows[str(M)] = row
        res[mode_name] = rows
        if model.device_status() != txs.TXS_OK:
            raise RuntimeError("device status after the sweep")
        cache.close()
        model.close()
    # appends of dL rows per request against the rebuild of all L rows
    model = txs.Model(base, weights, txs.LOCAL_GLOBAL)
    reps = 5
    cache = txs.KVCache(model, b0.beh_off, beh, capacity_extra=sum(SWEEP_DL) * (reps + 3))
    rng = np.random.default_rng(20268)
    app = {}
    for dL in SWEEP_DL:
        new = txs.to_device(W.round_bf16(rng.standard_normal((base.n_req * dL, d), dtype=np.float32)), dt)
        off = np.arange(base.n_req + 1, dtype=np.int32) * dL
        app[str(dL)] = timed(lambda: cache.append(off, new), reps, flush_l2=False)
    rebuild = timed(lambda: cache.rebuild(b0.beh_off, beh), 5)
    res["append_ms"] = app
    res["rebuild_ms"] = rebuild
    res["append_note"] = ("append: K/V projection of the new rows into their slots, pooling-state merge, anchor "
                          "re-projection; rebuild: the same for all L rows of every request (L2 flushed first)")
    if model.device_status() != txs.TXS_OK:
        raise RuntimeError("device status after the append sweep")
    cache.close()
    model.close()
    return res


DW_FIELDS = dict(dw_in=64, dw_out=32, dw_hidden=256)   # Deep & Wide head on the headline model


def deep_wide_bench(txs, torch):
    """The headline workload's score + rank with the Deep & Wide f_dec (App. B)
    in place of the linear one, against the same prebuilt caches: candidates/s
    and the per-class time of one call, next to the linear head's."""
    wl0 = W.WORKLOADS[DW_WORKLOAD]
    res = {"workload": f"{DW_WORKLOAD} with the Deep & Wide head (wide {DW_FIELDS['dw_in']} -> {DW_FIELDS['dw_out']}, "
                       f"deep FFN [z, x_deep] -> {DW_FIELDS['dw_hidden']} -> d - {DW_FIELDS['dw_out']})",
           "unit": "candidates/s"}
    flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
    for name, wl in (("linear_head", wl0), ("deep_wide_head", W.with_sizes(wl0, **DW_FIELDS))):
        b = W.batch(wl)
        dt = txs.torch_dtype(wl.dtype)
        model = txs.Model(wl, W.weights(wl), txs.LOCAL_GLOBAL)
        cache = txs.KVCache(model, b.beh_off, txs.to_device(b.beh, dt))
        cand = txs.to_device(b.cand, dt)
        ctx = txs.to_device(b.ctx.reshape(-1, wl.d_model), dt)
        n = int(b.cand_off[-1])
        ws = torch.empty(txs.workspace_bytes(model, wl.n_req, n), dtype=torch.uint8, device="cuda")
        lg = torch.empty((n, wl.n_actions), dtype=torch.float32, device="cuda")
        pr = torch.empty_like(lg)
        rk = torch.empty(n, dtype=torch.int32, device="cuda")

        def call():
            txs.score(model, cache, b.cand_off, cand, ctx, workspace=ws, out_logits=lg, out_probs=pr)
            txs.rank(b.cand_off, pr, wl.n_actions, 0, 0, out=rk)
        for _ in range(3):
            call()
        times = []
        for _ in range(20):
            flush.zero_()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record()
            call()
            e1.record()
            e1.synchronize()
            times.append(e0.elapsed_time(e1))
        txs.profile_enable(True)
        call()
        torch.cuda.synchronize()
        prof = txs.profile_collect()
        txs.profile_enable(False)
        if model.device_status() != txs.TXS_OK:
            raise RuntimeError("device status after the Deep & Wide measurement")
        ms = statistics.median(times)
        res[name] = {"ms_per_call": ms, "candidates_per_s": n / (ms / 1e3),
                     "kernels_ms": {k: v[0] for k, v in prof.items()}}
        cache.close()
        model.close()
    return res


ENC_WORKLOAD = "enc_mid_bf16"   # 64 users x 4096 tokens, d = 512, 2 layers, 8 new tokens per user
ENC_APPENDS, ENC_PROFILED = 24, 8
# FP32 FMA lanes per SM and the maximum SM clock (nominal): the ALU peak of a
# SIMT kernel is 152 SMs x 128 lanes x 2 flop x 2070 MHz.
ALU_FP32_TFLOPS = 152 * 128 * 2 * 2.070e9 / 1e12


def encoder_bench(txs, torch, peaks, peak_src, tokens=0):
    """Behavior encoder (Sec. 4.1.1; App. D incremental encoding) on the
    64-user x 4096-token workload: the incremental append of 8 new tokens per
    user (the nearline streaming update) and the full-stream build, with the
    roofline of each one's attention kernel and the oracle on a sample."""
    ew = W.ENC_WORKLOADS[ENC_WORKLOAD]
    if tokens:
        ew = W.with_sizes(ew, L=tokens)
    w = W.enc_weights(ew)
    b = W.enc_batch(ew)
    dt = txs.torch_dtype(ew.dtype)
    d, es = ew.d_model, 2 if ew.dtype == "bf16" else 4
    enc = txs.Encoder(ew, w)
    subj = txs.to_device(b.subj, dt)
    types = torch.from_numpy(b.types).to("cuda")
    sa = txs.to_device(b.subj_app, dt)
    ta = torch.from_numpy(b.types_app).to("cuda")
    n, na = int(b.off[-1]), int(b.app_off[-1])
    ws = torch.empty(enc.workspace_bytes(n), dtype=torch.uint8, device="cuda")
    phi = torch.empty((n, d), dtype=dt, device="cuda")
    new = torch.empty((na, d), dtype=dt, device="cuda")
    n_app = 3 + ENC_APPENDS + ENC_PROFILED
    cap = int(b.dL.max()) * n_app
    res = {"workload": f"{ENC_WORKLOAD}: {ew.n_req} users x {int(b.L[0])} tokens, d={d}, H={ew.n_heads}, "
                       f"F={ew.d_ff}, {ew.n_layers} layers, R={ew.n_rel}, full causal; append = "
                       f"{int(b.dL[0])} new tokens per user", "unit": "tokens/s"}

    def ev_time(fn):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record()
        fn()
        e1.record()
        e1.synchronize()
        return e0.elapsed_time(e1)

    # build (prefill of every stream); the state's allocation is inside the call
    builds = []
    for _ in range(2):
        st = None

        def mk():
            nonlocal st
            st = txs.EncState(enc, b.off, subj, types, capacity_extra=cap, workspace=ws, phi_out=phi)
        builds.append(ev_time(mk))
        st.close()
    txs.profile_enable(True)
    st = txs.EncState(enc, b.off, subj, types, capacity_extra=cap, workspace=ws, phi_out=phi)
    torch.cuda.synchronize()
    prof_b = txs.profile_collect()
    txs.profile_enable(False)
    # incremental appends against the growing state (inputs far larger than L2)
    call = lambda: st.append(b.app_off, sa, ta, workspace=ws, phi_out=new)
    for _ in range(3):
        call()
    hist0 = int(st.lengths().mean())
    times = [ev_time(call) for _ in range(ENC_APPENDS)]
    txs.profile_enable(True)
    lens_before = st.lengths().astype(np.int64)
    for _ in range(ENC_PROFILED):
        call()
    torch.cuda.synchronize()
    prof_a = txs.profile_collect()
    txs.profile_enable(False)
    if enc.device_status() != txs.TXS_OK:
        raise RuntimeError("device status after the encoder measurement")
    ms_app = statistics.median(times)
    # attention roofline of the append: each launch (one layer) reads every
    # visible key and value row once and the new rows' q and writes their output
    dL = b.dL.astype(np.int64)
    byts = 0.0
    for k in range(ENC_PROFILED):
        L_end = lens_before + (k + 1) * dL
        byts += ew.n_layers * (2 * float(L_end.sum()) * d * es + 2 * na * d * es)
    attn_ms, attn_n = prof_a.get("enc_attn", (0.0, 0))
    ach = byts / (attn_ms / 1e3) / 1e9 if attn_n else None
    res["append"] = {
        "ms_per_call": ms_app, "tokens_per_s": na / (ms_app / 1e3), "users_per_s": ew.n_req / (ms_app / 1e3),
        "history_tokens_per_user": f"{hist0} .. {int(st.lengths().mean())}",
        "kernels_ms_per_call": {k: v[0] / ENC_PROFILED for k, v in prof_a.items()},
        "launches_per_call": sum(v[1] for v in prof_a.values()) // ENC_PROFILED,
        "roofline_attn": {"bound": "hbm", "achieved": ach, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                          "frac": ach / peaks["hbm_gbs"] if ach else None, "traffic": None,
                          "kernel": "enc_attn", "peak_source": f"{peak_src} (copy)",
                          "algorithmic_per_launch_bytes": byts / attn_n if attn_n else None}}
    # build roofline of the attention: 4 flop per visible (query, key) pair per dim
    L = b.L.astype(np.int64)
    pairs = float((L * (L + 1) // 2).sum()) if ew.window == 0 else None
    fl = ew.n_layers * pairs * 4 * d
    bms, bn_ = prof_b.get("enc_attn", (0.0, 0))
    ach_b = fl / (bms / 1e3) / 1e12 if bms else None
    if ew.dtype == "bf16":   # enc_fa_kernel: tcgen05 MMAs for Q K^T and P V
        roof_b = {"bound": "tensor", "peak": peaks["bf16_tflops"], "peak_source": f"{peak_src} (burst)"}
    else:                    # enc_attn_kernel: FP32 FMAs on the CUDA cores
        roof_b = {"bound": "alu", "peak": ALU_FP32_TFLOPS,
                  "peak_source": "derived: 152 SMs x 128 FP32 lanes x 2 flop x 2070 MHz"}
    roof_b.update({"achieved": ach_b, "unit": "TFLOP/s", "frac": ach_b / roof_b["peak"] if ach_b else None,
                   "traffic": None, "kernel": "enc_attn", "algorithmic_flops_per_launch": fl / ew.n_layers})
    res["build"] = {
        "ms_per_call": statistics.median(builds), "tokens_per_s": n / (statistics.median(builds) / 1e3),
        "note": "includes the state's device allocation (cudaMalloc) inside the call",
        "kernels_ms": {k: v[0] for k, v in prof_b.items()},
        "roofline_attn": roof_b}
    st.close()
    enc.close()
    res["cpu_baseline"] = encoder_cpu_baseline(ew, w, b)
    return res


def encoder_cpu_baseline(ew, w, b, users=(0, 1), reps=20):
    """The encoder oracle as it stands on the host cores: the same append (8
    new tokens of a user with 4096 earlier ones) for a sample of users, the
    users' states built outside the timed region."""
    from oracle import encoder_oracle as E
    om = E.EncModel.from_arrays(w, ew)
    t_tot, toks = 0.0, 0
    for r in users:
        sl = slice(b.off[r], b.off[r + 1])
        _, st = E.encode(om, b.subj[sl], b.types[sl])
        sa = slice(b.app_off[r], b.app_off[r + 1])
        for _ in range(reps):
            t0 = time.perf_counter()
            E.encode_append(om, st, b.subj_app[sa], b.types_app[sa])
            t_tot += time.perf_counter() - t0
            toks += sa.stop - sa.start
    return {"value": float(toks / t_tot), "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle",
            "sample": f"append of {int(b.dL[0])} tokens for users {list(users)} of {ENC_WORKLOAD}, {reps} times "
                      f"each (float64 NumPy, {t_tot:.2f} s; the states are built outside the timing)"}


# ---------------------------------------------------------------- the oracle (CPU) arm

def oracle_step(O, model, wl, b, r):
    """One request through the oracle: cache build, append, scoring, ranking."""
    phi = b.beh[b.beh_off[r]:b.beh_off[r + 1]]
    c = O.build_cache(model, phi)
    c = O.append_cache(model, c, b.app[b.app_off[r]:b.app_off[r + 1]])
    _, pr = O.score_request(model, c, b.ctx[r], b.cand[b.cand_off[r]:b.cand_off[r + 1]])
    O.rank(pr[:, 0], [0, pr.shape[0]])
    return pr.shape[0]


def sample_requests(wl: W.Workload):
    """Requests of a bounded oracle sample: the shortest and the longest
    history first, then the others in a seeded order."""
    L, _, _ = W.sizes(wl)
    first = [int(np.argmin(L)), int(np.argmax(L))]
    rest = [int(r) for r in np.random.default_rng(wl.seed).permutation(wl.n_req) if int(r) not in first]
    return (first[:1] if first[0] == first[1] else first) + rest


def cpu_baseline(workload: str, budget_s: float, n_min: int = 8):
    """The oracle as it stands on the host cores: whole request-steps (cache
    build + append + score + rank) over at least n_min requests, the shortest
    and the longest history among them, until budget_s of work.  Candidates
    per second over the sample stand for the whole batch (extrapolated)."""
    from oracle import txs_oracle as O
    wl = W.WORKLOADS[workload]
    model = O.Model.from_arrays(W.weights(wl), wl)
    order = sample_requests(wl)
    n_done, cands, t_tot, seen = 0, 0, 0.0, []
    while n_done < min(n_min, wl.n_req) or t_tot < budget_s:
        r = order[n_done % len(order)]
        b = W.batch(wl, requests=[r])
        t0 = time.perf_counter()
        cands += oracle_step(O, model, wl, b, 0)
        t_tot += time.perf_counter() - t0
        seen.append((r, int(b.L[0])))
        n_done += 1
        if n_done >= 50 * wl.n_req:
            break
    Ls = [x[1] for x in seen]
    return {"value": cands / t_tot, "unit": "candidates/s", "cores": os.cpu_count(), "kind": "oracle",
            "sample": f"{n_done} request-steps over {len(set(x[0] for x in seen))} of the {wl.n_req} requests of "
                      f"{workload} (behavior lengths {min(Ls)}..{max(Ls)}, the batch's shortest and longest "
                      f"included), each cache build + append + score + rank in float64 NumPy ({t_tot:.1f} s); "
                      f"candidates/s over the sample, extrapolated to the batch"}


REF_TIME_CAP_S = 150.0


def run_reference(args, rank, world):
    """The oracle, as it stands, timed on the host cores: each step one whole
    request of the same workload (cache build + append + score + rank),
    cycling over the shortest, the longest and then seeded other requests;
    same metric, unit and config.  Stops early after REF_TIME_CAP_S of timed
    work so that a large --steps still ends within minutes."""
    from oracle import txs_oracle as O
    wl = W.WORKLOADS[args.workload]
    model = O.Model.from_arrays(W.weights(wl), wl)
    order = sample_requests(wl)
    batches = {}

    def get(i):
        r = order[i % len(order)]
        if r not in batches:
            batches[r] = W.batch(wl, requests=[r])
        return batches[r]
    for i in range(min(max(args.warmup, 1), 2)):
        oracle_step(O, model, wl, get(i), 0)
    cands, t_tot, done = 0, 0.0, 0
    for i in range(args.steps):
        b = get(i)
        t0 = time.perf_counter()
        cands += oracle_step(O, model, wl, b, 0)
        t_tot += time.perf_counter() - t0
        done += 1
        if t_tot > REF_TIME_CAP_S:
            break
    value = cands / t_tot
    reqs = [order[i % len(order)] for i in range(done)]
    Ls = [int(get(i).L[0]) for i in range(done)]
    sample = (f"{done} of {args.steps} steps{' (time cap reached)' if done < args.steps else ''}, each one whole "
              f"request of {args.workload} (requests {sorted(set(reqs))[:12]}{'...' if len(set(reqs)) > 12 else ''}, "
              f"behavior lengths {min(Ls)}..{max(Ls)}): cache build + append + score + rank in float64 NumPy on "
              f"the GPU box's host cores")
    return {"impl": "reference", "metric": METRIC, "value": value, "unit": "candidates/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * t_tot / done,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded N(0,1) inputs, N(0,0.02) weights; shapes of the paper's serving setting)",
            "config": step_config(wl, args.mode, world),
            "cpu_baseline": {"value": value, "unit": "candidates/s", "cores": os.cpu_count(), "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": "candidates/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def main():
    args = parse()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(run_reference(args, rank, world)), flush=True)
        return
    if args.section:
        import torch
        from paper_2607_28940_gb300 import build as B
        from paper_2607_28940_gb300 import txs
        B.build()
        peaks, peak_src = load_peaks()
        fn = {"encoder": lambda: encoder_bench(txs, torch, peaks, peak_src, args.enc_len),
              "deep_wide": lambda: deep_wide_bench(txs, torch),
              "sweep": lambda: sweep_bench(txs, torch, peaks, peak_src),
              "latency": lambda: latency_sweep(txs, torch),
              "events": lambda: events_bench(txs, torch)}[args.section]
        print(json.dumps({args.section: fn()}, default=float), flush=True)
        return
    if world > 1:
        import torch
        torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
        torch.distributed.init_process_group("nccl")
    out = run_txs(args, rank, world)
    if rank == 0:
        print(json.dumps(out), flush=True)
    if world > 1:
        import torch
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
