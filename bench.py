#!/usr/bin/env python3
"""Benchmark of the FlashVLA streaming action-decode step on GB300 (libfva).

Default workload: the pi0.5-shaped expert (18 layers, width 1024, 8 query heads /
1 KV head of 256, MLP 4096, action dim 32) with a 560-token prefix and a K=10 x
H=50 buffer at batch 1, synthetic seeded inputs.  A step is one fva_step: one
expert forward over the whole buffer, the per-chunk Euler update, emit, roll and
tail push.

Prints ONE JSON line (rank 0):
  value       steps/s with every input resident in HBM (CUDA-graph replay through
              fva_step, CUDA events on the launching stream, max over ranks);
  e2e         the same through the C ABI on pinned host buffers: every step's kernels
              read the action buffer from host memory and write the updated buffer
              and the emitted chunk back (e2e_copies: torch copies on the stream
              around the step on device buffers instead);
  roofline    the dominant kernel (largest share of a kernel-by-kernel profiled
              step) against the measured peak of its binding resource;
  step_roofline  the whole step against max(FLOPs / tensor peak, bytes / HBM peak);
  cpu_baseline   the CPU oracle timed on this host on a bounded sample.
Under torchrun every rank runs an independent replica (requests shard with no
exchange); `value` counts the steps of all ranks.

`--impl reference` times the CPU oracle instead (the reference arm).
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
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import workloads as WL  # noqa: E402

METRIC = "streaming decode steps/s (executable chunks/s) at batch 1; µs/step; % of roofline"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return p, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def dram_traffic(workload, kind):
    """DRAM bytes (read + write) per launch of `kind` from the committed ncu
    summary, if it was taken on this workload with the kernel's sources unchanged
    since (else None)."""
    path = os.path.join(ROOT, "profiles", "dram_traffic.json")
    try:
        with open(path) as f:
            tab = json.load(f)
    except (OSError, ValueError):
        return None
    e = tab.get(workload, {}).get(kind)
    if not e:
        return None
    sources = e.get("sources") or {e["source"]: e["source_sha256"]}
    for rel, want in sources.items():
        try:
            with open(os.path.join(ROOT, rel), "rb") as f:
                if hashlib.sha256(f.read()).hexdigest() != want:
                    return None
        except OSError:
            return None
    return e["dram_bytes_per_launch"]


# ---------------------------------------------------------------------------
# algorithmic work per kernel launch (FLOPs, bytes)
# ---------------------------------------------------------------------------

def kernel_costs(wl, B, n_sms=152):
    """Algorithmic FLOPs and DRAM bytes of one launch of each kernel kind (bf16
    weights, bf16 activations, fp32 residual stream)."""
    W, F, Dq, dh, nq, K, H, A = (wl.width, wl.mlp_dim, wl.n_q_heads * wl.head_dim,
                                 wl.head_dim, wl.n_q_heads, wl.n_chunks, wl.chunk_tokens,
                                 wl.action_dim)
    T = K * H
    M = B * T
    BK = B * K
    L = wl.n_layers
    Nqkv = Dq + 2 * dh
    Nmod = L * 6 * W + 2 * W
    P = wl.prefix_lens[:B]
    pairs = sum(p * T + H * H * K * (K + 1) // 2 for p in P)
    c = {}
    c["qkv"] = (2.0 * M * W * Nqkv, 2.0 * (Nqkv * W + M * W + M * Nqkv))
    c["out_proj"] = (2.0 * M * Dq * W, 2.0 * (W * Dq + M * Dq) + 4.0 * M * W)
    c["gate_up"] = (2.0 * M * W * 2 * F, 2.0 * (2 * F * W + M * W + M * F))
    c["down"] = (2.0 * M * F * W, 2.0 * (W * F + M * F) + 4.0 * M * W)
    c["attention"] = (4.0 * dh * nq * pairs, 2.0 * (sum(P) + B * T) * dh * 2 + 2.0 * 2 * M * Dq)
    c["film"] = (2.0 * BK * W * Nmod, 2.0 * Nmod * W + 4.0 * BK * Nmod)
    c["time_mlp"] = (2.0 * BK * W * W, 2.0 * W * W)
    c["resid_norm"] = (0.0, 4.0 * M * W * 3 + 2.0 * M * W)
    c["embed_norm"] = (2.0 * M * A * W, 4.0 * M * (A + W) + 2.0 * M * W)
    c["final_norm"] = (0.0, 4.0 * M * W * 3 + 4.0 * M * W)
    c["velocity"] = (2.0 * M * W * A, 4.0 * M * W + 4.0 * W * A + 4.0 * M * A * 3)
    tiles = -(-T * nq // 128)
    # the library's split of the key range: 1-4 blocks of 64 keys per split, the
    # largest that still gives about half as many attention CTAs as SMs
    nkb = -(-(max(P) + T) // 64)
    bps = 4
    while bps > 1 and B * tiles * -(-nkb // bps) < max(1, n_sms // 2):
        bps //= 2
    nsplit = -(-nkb // bps)
    # bf16 partial rows (O / l) and fp32 (max, sum) read, bf16 output written
    c["attn_merge"] = (0.0, (2.0 * dh + 8.0) * B * tiles * 128 * nsplit + 2.0 * M * Dq)
    c["timestep_embed"] = (0.0, 2.0 * BK * W)
    return c


def step_costs(wl, B, film=True):
    """Whole-step algorithmic FLOPs and the HBM bytes that must be streamed (every
    weight once + the prefix K/V of every layer).  film=False: the step that reuses
    the previous step's FiLM modulation (no time MLP, no FiLM projection)."""
    L = wl.n_layers
    c = kernel_costs(wl, B)
    flops = L * sum(c[k][0] for k in ("qkv", "out_proj", "gate_up", "down", "attention"))
    flops += c["embed_norm"][0] + c["velocity"][0]
    if film:
        flops += c["film"][0] + 2 * c["time_mlp"][0]
    W, F, Dq, dh, A = wl.width, wl.mlp_dim, wl.n_q_heads * wl.head_dim, wl.head_dim, wl.action_dim
    wbytes = 2.0 * L * ((Dq + 2 * dh) * W + W * Dq + 2 * F * W + W * F) + 4.0 * 2 * A * W
    if film:
        wbytes += 2.0 * (L * 6 * W + 2 * W) * W + 2.0 * 2 * W * W
    kv = 2.0 * L * sum(wl.prefix_lens[:B]) * dh * 2
    return flops, wbytes + kv


# ---------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.proc = None
        self.tmp = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(gpu_index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=self.tmp, stderr=subprocess.DEVNULL)
        except (OSError, ValueError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.tmp.flush()
        with open(self.tmp.name) as f:
            rows = [r.split(",") for r in f.read().strip().splitlines() if r.strip()]
        os.unlink(self.tmp.name)
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            r = [x.strip() for x in r]
            if len(r) < 7:
                continue
            try:
                sm.append(float(r[0]))
                mx = float(r[1])
            except ValueError:
                continue
            for n, v in zip(names, r[3:7]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


def gpu_index_for(local_rank: int) -> int:
    vis = os.environ.get("CUDA_VISIBLE_DEVICES")
    if vis:
        ids = [v.strip() for v in vis.split(",") if v.strip()]
        if local_rank < len(ids) and ids[local_rank].isdigit():
            return int(ids[local_rank])
    return local_rank


# ---------------------------------------------------------------------------
# CPU oracle timing (baseline / reference arm)
# ---------------------------------------------------------------------------

def time_oracle(wl, w, pre, buf, tau, budget_s: float, max_steps: int):
    import oracle
    fresh = np.zeros((wl.batch, wl.chunk_tokens, wl.action_dim), np.float32)
    t0 = time.perf_counter()
    oracle.stream_step(w, wl.as_config(), buf, tau, pre, fresh)
    first = time.perf_counter() - t0
    n = int(max(1, min(max_steps, budget_s // max(first, 1e-9))))
    t0 = time.perf_counter()
    for _ in range(n):
        oracle.stream_step(w, wl.as_config(), buf, tau, pre, fresh)
    dt = time.perf_counter() - t0
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    return n, dt, cores


_ORACLE_ONE_THREAD = r"""
import json, os, sys, time
sys.path.insert(0, sys.argv[1])
import numpy as np
import oracle
import workloads as WL
wl = WL.standard_workloads()[sys.argv[2]]
budget = float(sys.argv[3])
w = WL.make_weights(wl); pre = WL.make_prefix_kv(wl)
buf, tau = WL.make_buffer(wl), WL.make_noise_levels(wl)
fresh = np.zeros((wl.batch, wl.chunk_tokens, wl.action_dim), np.float32)
t0 = time.perf_counter(); oracle.stream_step(w, wl.as_config(), buf, tau, pre, fresh)
first = time.perf_counter() - t0
n = int(max(1, min(50, budget // max(first, 1e-9))))
t0 = time.perf_counter()
for _ in range(n):
    oracle.stream_step(w, wl.as_config(), buf, tau, pre, fresh)
print(json.dumps({"n": n, "dt": time.perf_counter() - t0}))
"""


def time_oracle_one_thread(wl_name: str, budget_s: float):
    """The oracle on one host core: a child process with every BLAS / OpenMP thread
    pool limited to one thread (set before NumPy loads)."""
    env = dict(os.environ, OPENBLAS_NUM_THREADS="1", OMP_NUM_THREADS="1", MKL_NUM_THREADS="1",
               BLIS_NUM_THREADS="1", NUMEXPR_NUM_THREADS="1", CUDA_VISIBLE_DEVICES="")
    try:
        out = subprocess.run([sys.executable, "-c", _ORACLE_ONE_THREAD, ROOT, wl_name,
                              str(budget_s)], env=env, capture_output=True, text=True,
                             timeout=20 * budget_s + 120)
        r = json.loads(out.stdout.strip().splitlines()[-1])
        return r["n"], r["dt"]
    except (OSError, ValueError, IndexError, KeyError, subprocess.TimeoutExpired):
        return None


# ---------------------------------------------------------------------------
# isolated chunk-causal attention over the prefix sweep (T = 500 action tokens)
# ---------------------------------------------------------------------------

def attention_sweep(dev, stream, peaks, prefixes=(256, 512, 1024, 2048, 4096), iters=40):
    """fva_chunk_attention on one layer's inputs (K=10 x H=50 tokens, 8 query heads of
    256, one KV head) for each prefix length P.  Every launch reads a different copy
    of K and V, and the copies together exceed the 129 MB L2, so the prefix keys come
    from HBM as in the step; q (written just before attention in the step) is one
    copy.  CUDA events on the launching stream."""
    import torch
    import paper_2608_27384_gb300 as fva
    from paper_2608_27384_gb300.harness import config_for
    K, H, nq, dh = 10, 50, 8, 256
    T = K * H
    wl = WL.small_bf16_workload(n_layers=1, n_q_heads=nq, n_chunks=K, chunk_tokens=H,
                                prefix_lens=[max(prefixes)])
    h = fva.fva_create(config_for(wl))
    out_rows = []
    try:
        gen = torch.Generator(device=dev).manual_seed(0)
        q = torch.randn((T * nq, dh), device=dev, generator=gen).to(torch.bfloat16)
        o = torch.empty_like(q)
        for P in prefixes:
            kv_rows = P + T
            per_copy = 2 * kv_rows * dh * 2
            n_copy = max(2, -(-160 * 2 ** 20 // per_copy))
            kp = torch.randn((n_copy, kv_rows, dh), device=dev, generator=gen).to(torch.bfloat16)
            vp = torch.randn((n_copy, kv_rows, dh), device=dev, generator=gen).to(torch.bfloat16)
            pl = torch.tensor([P], dtype=torch.int32, device=dev)
            with torch.cuda.stream(stream):
                for i in range(3):
                    fva.fva_chunk_attention(h, q, kp[i % n_copy], vp[i % n_copy], pl, 1, kv_rows,
                                            o, stream)
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                for i in range(iters):
                    fva.fva_chunk_attention(h, q, kp[i % n_copy], vp[i % n_copy], pl, 1, kv_rows,
                                            o, stream)
                e1.record(stream)
            torch.cuda.synchronize()
            us = 1e3 * e0.elapsed_time(e1) / iters
            pairs = P * T + H * H * K * (K + 1) // 2
            flops = 4.0 * dh * nq * pairs
            tf = flops / (us * 1e-6) / 1e12
            out_rows.append({"prefix": P, "us": round(us, 3), "tflops": round(tf, 1),
                             "frac_of_burst": round(tf / peaks["bf16_tflops"], 4),
                             "kv_copies": n_copy})
            del kp, vp
    finally:
        fva.fva_destroy(h)
    return out_rows


def ncu_launch_shares(workload):
    """Per-kind shares of the committed ncu launch list of this workload, if any."""
    path = os.path.join(ROOT, "profiles", f"step_{workload}_launches.json")
    try:
        with open(path) as f:
            return json.load(f)
    except (OSError, ValueError):
        return None


# ---------------------------------------------------------------------------

class Replicas:
    """The multi-GPU form of the step: independent replicas, one per rank (requests
    shard by rank; no collective on the data path).  The only cross-rank traffic
    is the harness's barrier around the timed region and the max over ranks of
    its duration.  backend "nccl" on GPUs; "gloo" serves the CPU tests."""

    def __init__(self, world: int, backend: str, device):
        import torch
        self.torch = torch
        self.device = device
        self.dist = None
        if world > 1:
            import torch.distributed as dist
            if backend == "nccl":
                dist.init_process_group(backend, device_id=device)
            else:
                dist.init_process_group(backend)
            self.dist = dist

    def _sync(self):
        if self.device.type == "cuda":
            self.torch.cuda.synchronize(self.device)

    def barrier(self):
        self._sync()
        if self.dist is not None:
            self.dist.barrier()
        self._sync()

    def max(self, x: float) -> float:
        if self.dist is None:
            return x
        t = self.torch.tensor([x], device=self.device, dtype=self.torch.float64)
        self.dist.all_reduce(t, op=self.dist.ReduceOp.MAX)
        return float(t.item())

    def close(self):
        if self.dist is not None:
            self.dist.destroy_process_group()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=4000)
    ap.add_argument("--warmup", type=int, default=50)
    ap.add_argument("--impl", choices=["fva", "reference"], default="fva")
    ap.add_argument("--workload", default="pi05_2view", choices=list(WL.standard_workloads()))
    ap.add_argument("--profile-steps", type=int, default=20)
    ap.add_argument("--cpu-budget", type=float, default=20.0,
                    help="seconds of oracle work for the CPU baseline")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-isolated", action="store_true",
                    help="skip the isolated-decode comparison (K passes over one chunk)")
    ap.add_argument("--no-sweep", action="store_true",
                    help="skip the isolated attention prefix sweep")
    ap.add_argument("--clock-soak", type=float, default=1.5,
                    help="seconds of untimed steps before the timed region while clocks are sampled")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    wl = WL.standard_workloads()[args.workload]
    peaks, peak_src = load_peaks()
    cfg_json = {"workload": wl.name, "batch": wl.batch, "n_chunks": wl.n_chunks,
                "chunk_tokens": wl.chunk_tokens, "prefix_tokens": wl.prefix_lens[:4],
                "n_layers": wl.n_layers, "width": wl.width, "heads": f"{wl.n_q_heads}q/1kv",
                "head_dim": wl.head_dim, "mlp_dim": wl.mlp_dim, "action_dim": wl.action_dim,
                "parallelism": f"replicas x{args.gpus}" if args.gpus > 1 else "single GPU",
                "l2": "no flush: every step streams ~0.87 GB of weights + prefix K/V > 129 MB L2",
                "weights": "seeded N(0, 0.02), bf16"}

    if args.impl == "reference":
        if rank != 0:
            return 0
        import oracle
        w = WL.make_weights(wl)
        pre = WL.make_prefix_kv(wl)
        buf, tau = WL.make_buffer(wl), WL.make_noise_levels(wl)
        fresh = np.zeros((wl.batch, wl.chunk_tokens, wl.action_dim), np.float32)
        step = lambda: oracle.stream_step(w, wl.as_config(), buf, tau, pre, fresh)  # noqa: E731
        # --warmup untimed steps, then --steps timed ones; if that would take more than
        # about four minutes, as many of each as fit (the line reports the counts used)
        t0 = time.perf_counter()
        step()
        first = time.perf_counter() - t0
        fit = max(2, int(240.0 // max(first, 1e-9)))
        n_warm = max(1, min(args.warmup, fit // 4))
        n = max(1, min(args.steps, fit - n_warm))
        for _ in range(n_warm - 1):
            step()
        t0 = time.perf_counter()
        for _ in range(n):
            step()
        dt = time.perf_counter() - t0
        cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
        v = n / dt
        line = {"metric": METRIC, "value": v, "unit": "steps/s", "impl": "reference",
                "n_gpus": args.gpus, "steps": n, "warmup": n_warm, "ms_per_step": 1e3 * dt / n,
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
                "dtype": "f64", "data": "synthetic", "config": cfg_json,
                "cpu_baseline": {"value": v, "unit": "steps/s", "cores": cores, "kind": "oracle",
                                 "sample": f"{n} timed full oracle steps after {n_warm} untimed "
                                           f"(requested {args.steps} and {args.warmup}; bounded "
                                           "to ~4 min of CPU work)"},
                "e2e": {"value": v, "unit": "steps/s", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}}
        print(json.dumps(line))
        return 0

    import torch
    import paper_2608_27384_gb300 as fva
    from paper_2608_27384_gb300.harness import Decoder

    torch.cuda.set_device(local_rank if world > 1 else 0)
    dev = torch.device("cuda", local_rank if world > 1 else 0)
    replicas = Replicas(world, "nccl", dev)

    w = WL.make_weights(wl)
    pre = WL.make_prefix_kv(wl)
    buf = WL.make_buffer(wl)
    tau = WL.make_noise_levels(wl)
    dec = Decoder(wl, WL.flat_weights(wl, w), pre)
    h = dec.handle
    B = wl.batch
    stream = torch.cuda.Stream(device=dev)
    d_buf = torch.from_numpy(buf).to(dev)
    d_out = torch.empty((B, wl.chunk_tokens, wl.action_dim), device=dev)

    barrier = replicas.barrier
    max_over_ranks = replicas.max

    # ---- device-resident timing: graph replay through fva_step
    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            fva.fva_step(h, d_buf, tau, d_out, B, stream)
    torch.cuda.synchronize(dev)
    # The clocks are sampled every 200 ms from here to the end of the timed region.  A
    # timed region of a few steps lasts milliseconds, so untimed steps (the clock
    # soak, not counted anywhere) keep the GPU under the same load for about 1.5 s
    # before it and the samples describe the clocks the timed steps ran at.
    sampler = ClockSampler(gpu_index_for(local_rank))
    soak_steps = 0
    soak_t0 = time.perf_counter()
    with torch.cuda.stream(stream):
        while time.perf_counter() - soak_t0 < args.clock_soak:
            for _ in range(100):
                fva.fva_step(h, d_buf, tau, d_out, B, stream)
            soak_steps += 100
            stream.synchronize()
    barrier()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(args.steps):
        fva.fva_step(h, d_buf, tau, d_out, B, stream)
    ev1.record(stream)
    barrier()
    clocks = sampler.stop()
    ms = max_over_ranks(ev0.elapsed_time(ev1))
    steps_total = args.steps * world
    value = steps_total / (ms / 1e3)
    us_per_step = 1e3 * ms / args.steps

    # ---- end to end: the C-ABI step on pinned HOST buffers.  Every step's kernels read
    # the action buffer from host memory (the in-projection and the Euler update each
    # read it), write the updated buffer and the emitted chunk back to host memory,
    # and take tau / dt from the pinned parameter ring: all transfers happen inside
    # the timed steps, over the host link, with no copy queued on the stream.
    h_buf = torch.from_numpy(buf).pin_memory()
    h_out = torch.empty((B, wl.chunk_tokens, wl.action_dim)).pin_memory()
    e2e_steps = max(10, args.steps // 4)
    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            fva.fva_step(h, h_buf, tau, h_out, B, stream)
        barrier()
        ev0.record(stream)
        for _ in range(e2e_steps):
            fva.fva_step(h, h_buf, tau, h_out, B, stream)
        ev1.record(stream)
    barrier()
    e2e_ms = max_over_ranks(ev0.elapsed_time(ev1))
    e2e_value = e2e_steps * world / (e2e_ms / 1e3)
    h2d = 2 * buf.nbytes + tau.nbytes
    d2h = buf.nbytes + h_out.numel() * 4
    # the same through copies queued on the stream around the step on device buffers
    # (pinned buffer in, emitted chunk out): context for the number above
    e2e_copies = None
    if rank == 0:
        with torch.cuda.stream(stream):
            for _ in range(args.warmup):
                d_buf.copy_(h_buf, non_blocking=True)
                fva.fva_step(h, d_buf, tau, d_out, B, stream)
                h_out.copy_(d_out, non_blocking=True)
            ec0 = torch.cuda.Event(enable_timing=True)
            ec1 = torch.cuda.Event(enable_timing=True)
            ec0.record(stream)
            for _ in range(e2e_steps):
                d_buf.copy_(h_buf, non_blocking=True)
                fva.fva_step(h, d_buf, tau, d_out, B, stream)
                h_out.copy_(d_out, non_blocking=True)
            ec1.record(stream)
        torch.cuda.synchronize()
        e2e_copies = {"value": e2e_steps / (ec0.elapsed_time(ec1) / 1e3), "unit": "steps/s",
                      "h2d_bytes_per_step": buf.nbytes, "d2h_bytes_per_step": h_out.numel() * 4,
                      "note": "torch copies on the stream around fva_step on device buffers"}

    # ---- the same step reusing the previous step's FiLM modulation (steady streaming
    # keeps the noise levels fixed, §3.2): a separately labelled extra number
    film_cached = None
    if rank == 0:
        with torch.cuda.stream(stream):
            for _ in range(args.warmup):
                fva.fva_step_ex(h, d_buf, tau, d_out, B, reuse_film=True, stream=stream)
            ec0 = torch.cuda.Event(enable_timing=True)
            ec1 = torch.cuda.Event(enable_timing=True)
            ec0.record(stream)
            for _ in range(args.steps):
                fva.fva_step_ex(h, d_buf, tau, d_out, B, reuse_film=True, stream=stream)
            ec1.record(stream)
        torch.cuda.synchronize()
        us_c = 1e3 * ec0.elapsed_time(ec1) / args.steps
        fl_c, by_c = step_costs(wl, B, film=False)
        roof_c = max(fl_c / (peaks["bf16_tflops"] * 1e12), by_c / (peaks["hbm_gbs"] * 1e9))
        film_cached = {"us_per_step": us_c, "steps_per_s": 1e6 / us_c,
                       "roofline_us": 1e6 * roof_c, "frac": 1e6 * roof_c / us_c,
                       "note": "FVA_STEP_REUSE_FILM: the time MLP and FiLM projections of the "
                               "previous step are reused (noise levels unchanged); not the "
                               "headline, which recomputes them every step"}

    # ---- the same step with every layer's FiLM modulation computed before the first
    # layer (FVA_STEP_SERIAL_FILM; the default computes layer 0's scale / shift first
    # and the rest in the QKV projections' launches): the comparison, and the baseline
    # of the per-launch event-node cost below (the profiled step computes the FiLM
    # the same way)
    film_serial = None
    if rank == 0:
        with torch.cuda.stream(stream):
            for _ in range(args.warmup):
                fva.fva_step_ex(h, d_buf, tau, d_out, B, serial_film=True, stream=stream)
            es0 = torch.cuda.Event(enable_timing=True)
            es1 = torch.cuda.Event(enable_timing=True)
            es0.record(stream)
            for _ in range(args.steps):
                fva.fva_step_ex(h, d_buf, tau, d_out, B, serial_film=True, stream=stream)
            es1.record(stream)
        torch.cuda.synchronize()
        us_s = 1e3 * es0.elapsed_time(es1) / args.steps
        film_serial = {"us_per_step": us_s, "steps_per_s": 1e6 / us_s,
                       "note": "FVA_STEP_SERIAL_FILM: every layer's FiLM modulation computed "
                               "before the first layer; the headline computes it in the QKV "
                               "projections' launches (same bits)"}

    # ---- kernel-by-kernel profile (CUDA events between launches on `stream`)
    per_kind = {}
    launches_per_step = 0
    for _ in range(args.profile_steps):
        recs = fva.fva_step_profile(h, d_buf, tau, d_out, B, stream)
        launches_per_step = len(recs)
        for kind, _layer, us in recs:
            t, n = per_kind.get(kind, (0.0, 0))
            per_kind[kind] = (t + us, n + 1)
    prof_total = sum(t for t, _ in per_kind.values())
    costs = kernel_costs(wl, B, torch.cuda.get_device_properties(dev).multi_processor_count)
    bw = peaks["hbm_gbs"] * 1e9
    tc = peaks["bf16_tflops"] * 1e12
    # The event nodes serialise the profiled graph and add a fixed cost to every
    # launch: (profiled step - timed step) / launches, spread evenly, is taken off
    # each launch (never more than 3/4 of it).  The profiled step computes the FiLM
    # modulation before the first layer, so the timed step it is compared with is
    # the one that does the same.
    prof_step_us = prof_total / max(1, args.profile_steps)
    base_us = film_serial["us_per_step"] if film_serial else us_per_step
    overhead_us = max(0.0, (prof_step_us - base_us) / max(1, launches_per_step))
    corr = {k: (max(t - n * overhead_us, 0.25 * t), n) for k, (t, n) in per_kind.items()}
    dom = max(corr, key=lambda k: corr[k][0])
    t_us, n = corr[dom]
    avg_s = t_us / n * 1e-6
    fl, by = costs[dom]
    if fl / tc >= by / bw:
        # the kernel is timed inside the step loop: the sustained tensor peak
        roof = {"bound": "tensor", "achieved": fl / avg_s / 1e12,
                "peak": peaks["bf16_tflops_sustained"], "unit": "TFLOP/s"}
    else:
        roof = {"bound": "hbm", "achieved": by / avg_s / 1e9, "peak": peaks["hbm_gbs"],
                "unit": "GB/s"}
    roof["frac"] = roof["achieved"] / roof["peak"]
    if roof["bound"] == "tensor":
        roof["frac_of_burst"] = roof["achieved"] / peaks["bf16_tflops"]
    roof.update({"traffic": dram_traffic(args.workload, dom), "kernel": dom,
                 "launches_per_step": n // max(1, args.profile_steps),
                 "avg_launch_us": t_us / n, "avg_launch_us_with_event_nodes": per_kind[dom][0] / n,
                 "event_node_overhead_us": overhead_us,
                 "share_of_step": t_us / max(1, args.profile_steps) / us_per_step,
                 "peak_source": f"{peak_src} " + ("sustained" if roof["bound"] == "tensor"
                                                  else "copy")})
    per_kind = corr
    prof_total = sum(t for t, _ in per_kind.values())
    shares = {k: round(v[0] / prof_total, 4) for k, v in sorted(per_kind.items(),
                                                                key=lambda kv: -kv[1][0])}
    # every kernel kind against its own binding peak (same event-timed launches)
    kernel_rooflines = {}
    for k, (t_k, n_k) in per_kind.items():
        if k not in costs:
            continue
        fl_k, by_k = costs[k]
        avg_k = t_k / n_k * 1e-6
        tensor = fl_k / tc >= by_k / bw
        ach = (fl_k / avg_k / 1e12) if tensor else (by_k / avg_k / 1e9)
        kernel_rooflines[k] = {"bound": "tensor" if tensor else "hbm",
                               "avg_launch_us": round(t_k / n_k, 3),
                               "achieved": round(ach, 2),
                               "unit": "TFLOP/s" if tensor else "GB/s",
                               "frac": round(ach / (peaks["bf16_tflops_sustained"] if tensor
                                                    else peaks["hbm_gbs"]), 4)}

    flops, nbytes = step_costs(wl, B)
    t_roof = max(flops / tc, nbytes / bw)
    step_roof = {"flops": flops, "bytes": nbytes, "t_tensor_us": 1e6 * flops / tc,
                 "t_hbm_us": 1e6 * nbytes / bw, "roofline_us": 1e6 * t_roof,
                 "frac": 1e6 * t_roof / us_per_step,
                 "bound": "tensor" if flops / tc >= nbytes / bw else "hbm",
                 "peaks": f"{peak_src}: {peaks['bf16_tflops']} TFLOP/s bf16 burst, "
                          f"{peaks['hbm_gbs']} GB/s"}

    # The decode FlashVLA replaces (§1, App. A.3): pi0.5-style isolated denoising of
    # one chunk, K passes of the same expert over [prefix ; one chunk] per emitted
    # chunk.  Timed with the same graph replay on a K = 1 buffer of this expert.
    isolated = None
    if rank == 0 and wl.dtype == "bf16" and not args.no_isolated:
        wl1 = WL.Workload(**dict(wl.__dict__, name=wl.name + "_isolated", n_chunks=1))
        dec1 = Decoder(wl1, WL.flat_weights(wl1, w), pre)
        b1 = torch.from_numpy(WL.make_buffer(wl1)).to(dev)
        o1 = torch.empty((B, wl.chunk_tokens, wl.action_dim), device=dev)
        tau1 = np.full((B, 1), 1.0 / wl.n_chunks, dtype=np.float32)
        n1 = max(50, args.steps // 4)
        with torch.cuda.stream(stream):
            for _ in range(args.warmup):
                fva.fva_step(dec1.handle, b1, tau1, o1, B, stream)
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for _ in range(n1):
                fva.fva_step(dec1.handle, b1, tau1, o1, B, stream)
            e1.record(stream)
        torch.cuda.synchronize()
        us1 = 1e3 * e0.elapsed_time(e1) / n1
        dec1.close()
        isolated = {"passes_per_chunk": wl.n_chunks, "us_per_pass": us1,
                    "us_per_chunk": wl.n_chunks * us1, "streaming_us_per_chunk": us_per_step,
                    "speedup": wl.n_chunks * us1 / us_per_step,
                    "note": "K passes of the same expert over [prefix ; one chunk] per emitted "
                            "chunk (pi0.5-style decode), against one streaming step"}

    sweep = None
    if rank == 0 and wl.dtype == "bf16" and not args.no_sweep:
        sweep = attention_sweep(dev, stream, peaks)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        n_cpu, dt_cpu, cores = time_oracle(wl, w, pre, buf, tau, budget_s=args.cpu_budget,
                                           max_steps=1000)
        cpu = {"value": n_cpu / dt_cpu, "unit": "steps/s", "cores": cores, "kind": "oracle",
               "sample": f"{n_cpu} full oracle steps of the same workload (fp64 NumPy, BLAS "
                         f"threads on all {cores} host cores)"}
        one = time_oracle_one_thread(wl.name, args.cpu_budget / 2)
        if one is not None:
            cpu["single_thread"] = {"value": one[0] / one[1], "unit": "steps/s", "cores": 1,
                                    "sample": f"{one[0]} full oracle steps, every BLAS / OpenMP "
                                              "pool at one thread"}

    dec.close()
    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": "steps/s", "n_gpus": args.gpus,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms / args.steps,
                "us_per_step": us_per_step, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "bf16", "data": "synthetic", "config": cfg_json,
                "clocks": clocks,
                "e2e": {"value": e2e_value, "unit": "steps/s", "h2d_bytes_per_step": h2d,
                        "d2h_bytes_per_step": d2h, "steps": e2e_steps,
                        "api": "fva_step on pinned host buffers (the step's kernels read and "
                               "write host memory over the host link)"},
                "e2e_copies": e2e_copies,
                "gpu_launches": launches_per_step * args.steps,
                "roofline": roof, "step_roofline": step_roof, "kernel_shares": shares,
                "kernel_rooflines": kernel_rooflines,
                "profile_note": "per-kernel times: CUDA events between the kernels of a "
                                "captured profiling graph; the event nodes serialise the "
                                "kernels and cost about the same per launch, so "
                                "(profiled step - timed step with the FiLM computed first, "
                                "film_serial) / launches is taken off every launch "
                                "(roofline.event_node_overhead_us)",
                "isolated_decode": isolated,
                "attention_sweep": sweep,
                "film_cached": film_cached,
                "film_serial": film_serial,
                "ncu_launch_shares": ncu_launch_shares(args.workload),
                "clock_soak": {"steps": soak_steps, "seconds": args.clock_soak,
                               "note": "untimed steps between the warm-up and the timed "
                                       "region, under the clock sampler"},
                "cpu_baseline": cpu}
        print(json.dumps(line))
    replicas.close()
    return 0


if __name__ == "__main__":
    sys.exit(main())
