"""Benchmark of the thresholded gated-MLP decode path on one GB300.

Workload (by what it is): one Llama-3.1-8B-shaped MLP block (hidden 4096,
intermediate 14336), bf16 weights ~ N(0, 0.02), one decode token x ~ N(0, 1)
in bf16, thresholds t_l from 256 seeded calibration vectors (Eq. 3) at 50 %,
70 % and 90 % target sparsity.  One step = three sats_sparse_mlp calls, one
per sparsity level, each writing y and the compacted active-index list.
Each call reads a different one of four device copies of the layer, so a copy
is reused only after >= 420 MB of other weights have streamed (inputs larger
than the 129 MB L2).

The line also carries, under "batched", the same layer at decode-batch and
prefill sizes (8, 64, 256 and 2048 tokens per call, 50 % threshold), which run
on the tensor-core path: microseconds per call, tokens/s, weight-stream GB/s
and dense-equivalent TFLOP/s against the measured bf16 peak; and, under
"configs", the other four workloads at full size (the small layer, the
32-block Llama stack, the 36-block routed Qwen stack at 1 / 8 / 32 / 64 tokens
per step, the routed prefill block at 256 / 2048 tokens and 40 / 90 %), with
thresholds from the library's own Eq. 3 kernels.  The CPU oracle is timed on
one core and over all host cores (threshold recipe as the GPU arm: 256
calibration vectors).

Prints one JSON line.  `--impl reference` times the CPU oracle instead (the
reference arm of this comparison), on a bounded sample of the same workload,
one decode token per host core at a time.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2607_08991_gb300 import inputs  # noqa: E402

WORKLOAD = "llama_layer_4096x14336_b1"
SPARSITY = (0.5, 0.7, 0.9)
METRIC = "MLP decode us/token & achieved HBM GB/s vs peak at 50/70/90% sparsity"
LAYER_COPIES = 4
N_CALIB = 256
FUSED_SRC = os.path.join(ROOT, "paper_2607_08991_gb300", "csrc", "fused_mlp.cu")
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "fused_mlp_llama_layer_b1.md")
NOMINAL_HBM_GBS = 8000.0
BATCHES = (8, 64, 256, 2048)


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            pk = json.load(f)
        return float(pk["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def _bf16_peak():
    """Dense bf16 tensor peak (TFLOP/s): the measured burst figure, else the fallback."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["bf16_tflops"]), "measured"
    except Exception:
        return 1900.0, "fallback"


def _src_hash(path):
    with open(path, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


def _ncu_traffic():
    """DRAM bytes per launch from the committed ncu summary, if it was taken on this kernel source."""
    try:
        lines = open(TRAFFIC_FILE).read().splitlines()
    except OSError:
        return None
    vals = {}
    for ln in lines:
        if ":" in ln and ln.strip().startswith("- "):
            k, v = ln.strip()[2:].split(":", 1)
            vals[k.strip()] = v.strip().strip("`")
    if vals.get("kernel_source_sha256_16") != _src_hash(FUSED_SRC):
        return None
    try:
        return {s: float(vals["dram_bytes_per_launch_s%d" % int(round(100 * s))]) for s in SPARSITY}
    except (KeyError, ValueError):
        return None


class Clocks:
    """Samples SM clocks and throttle reasons with nvidia-smi during the timed region."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, local: int):
        vis = [v.strip() for v in os.environ.get("CUDA_VISIBLE_DEVICES", "").split(",") if v.strip()]
        self.index = vis[local] if local < len(vis) else str(local)
        self.proc = None
        self.path = os.path.join("/tmp", "sats_clocks_%d_%d.csv" % (os.getpid(), local))

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", self.index, "--query-gpu=" + self.QUERY,
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        try:
            for ln in open(self.path):
                f = [c.strip() for c in ln.split(",")]
                if len(f) < 9:
                    continue
                try:
                    sm.append(float(f[1]))
                    mx.append(float(f[2]))
                except ValueError:
                    continue
                for n, v in zip(names, f[5:9]):
                    if v.lower().startswith("active"):
                        reasons.add(n)
        finally:
            try:
                os.unlink(self.path)
            except OSError:
                pass
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "reasons": sorted(reasons)}


def _dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def _max_over_ranks(values, world: int, device=None):
    """Each value's maximum over the ranks of the default process group: the replicas run
    independently, and the job takes as long as the slowest."""
    if world <= 1:
        return [float(v) for v in values]
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(v) for v in t]


def _us_per_token(total_ms: float, steps: int, calls: int, world: int) -> float:
    """Whole-job time per token: each of `world` replicas runs steps x calls one-token calls
    in total_ms (the slowest replica's time)."""
    return total_ms * 1e3 / (steps * calls * world)


# ---------------------------------------------------------------------------- CPU oracle arm
def _headline_config(world: int):
    """The headline workload's config, shared by the GPU arm and the oracle arm."""
    H, N = inputs.LLAMA_H, inputs.LLAMA_N
    return {"workload": WORKLOAD, "hidden": H, "intermediate": N, "tokens": 1, "sparsity": list(SPARSITY),
            "calibration_vectors": N_CALIB,
            "l2": "inputs larger than L2: %d rotating device copies of the layer (%.2f GB)"
                  % (LAYER_COPIES, LAYER_COPIES * 6.0 * H * N / 1e9),
            "parallelism": "replicas" if world > 1 else "single"}


def _host_threads() -> int:
    try:
        return max(1, len(os.sched_getaffinity(0)))
    except AttributeError:
        return max(1, os.cpu_count() or 1)


def _oracle_setup():
    """The oracle's inputs for the headline workload: the layer, decode tokens, and the Eq. 3
    thresholds at 50 / 70 / 90 % from the same 256 calibration vectors the GPU arm uses (their
    gate activations computed on a thread pool over the host cores; setup, not timed)."""
    import concurrent.futures

    import oracle
    oracle.build()
    H, N = inputs.LLAMA_H, inputs.LLAMA_N
    w = inputs.mlp_weights(H, N)
    cal = oracle.bf16_to_f64(inputs.activations_bf16(N_CALIB, H, seed=inputs.SEED_CALIB))
    with concurrent.futures.ThreadPoolExecutor(_host_threads()) as ex:   # the C oracle releases the GIL
        parts = list(ex.map(lambda c: oracle.gate_act(cal[c:c + 4], w.Wg), range(0, N_CALIB, 4)))
    a_cal = np.concatenate(parts)
    ts = [oracle.percentile_threshold(a_cal, s) for s in SPARSITY]
    return oracle, w, ts


def _oracle_one_core(orc, w, ts, budget_s: float, max_calls: int = 64):
    """The oracle on one core: one token through the layer per call, sparsity levels cycling."""
    x = orc.bf16_to_f64(inputs.activations_bf16(1, inputs.LLAMA_H))
    times = []
    t_all = time.perf_counter()
    i = 0
    while i < max_calls and (i < len(SPARSITY) or time.perf_counter() - t_all < budget_s):
        t0 = time.perf_counter()
        orc.sparse_mlp(x, w.Wg, w.Wu, w.Wd, ts[i % len(SPARSITY)])
        times.append(time.perf_counter() - t0)
        i += 1
    us = 1e6 * sum(times) / len(times)
    sample = ("%d single-token calls on one core (hidden 4096, intermediate 14336, thresholds at %s sparsity "
              "from 256 calibration vectors)" % (len(times), "/".join(str(s) for s in SPARSITY)))
    return us, sample


def _oracle_all_cores(orc, w, ts, rounds: int, threads: int):
    """The oracle over the host cores: `threads` decode tokens at a time, one per thread (the C
    oracle releases the GIL), sparsity levels cycling over the tokens; us per token of wall time."""
    import concurrent.futures
    T = rounds * threads
    xs = orc.bf16_to_f64(inputs.activations_bf16(T, inputs.LLAMA_H, seed=inputs.SEED_X + 9))
    with concurrent.futures.ThreadPoolExecutor(threads) as ex:
        t0 = time.perf_counter()
        list(ex.map(lambda i: orc.sparse_mlp(xs[i:i + 1], w.Wg, w.Wu, w.Wd, ts[i % len(SPARSITY)]), range(T)))
        el = time.perf_counter() - t0
    return 1e6 * el / T, el


def run_reference(args):
    world, rank, _ = _dist_env()
    if rank != 0:
        return
    orc, w, ts = _oracle_setup()
    threads = _host_threads()
    # one step = one decode token per host core, all at once (sparsity levels cycling); a bounded sample
    _oracle_all_cores(orc, w, ts, max(args.warmup, 1), threads)
    us, el = _oracle_all_cores(orc, w, ts, args.steps, threads)
    sample = ("%d steps of %d single-token calls in parallel (one per host core), sparsity cycling %s, thresholds "
              "from 256 calibration vectors" % (args.steps, threads, "/".join(map(str, SPARSITY))))
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": us, "unit": "us/token", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * el / args.steps,
        "higher_is_better": False, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": _headline_config(world),
        "cpu_baseline": {"value": us, "unit": "us/token", "cores": threads, "kind": "oracle", "sample": sample},
        "e2e": {"value": us, "unit": "us/token", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


# ---------------------------------------------------------------------------- GPU arm
def run_gpu(args):
    import torch
    import torch.distributed as dist

    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_08991_gb300 import sats

    world, rank, local = _dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)

    H, N = inputs.LLAMA_H, inputs.LLAMA_N
    stream = torch.cuda.Stream(device=dev)
    w = inputs.mlp_weights(H, N)
    copies = 1 if (args.profile or args.profile_batch) else LAYER_COPIES
    with torch.cuda.stream(stream):
        src = [torch.from_numpy(m.view(np.int16)).to(dev) for m in (w.Wg, w.Wu, w.Wd)]
        layers = [sats.Layer(*src, stream=stream) for _ in range(copies)]
        del src
        ws = sats.Workspace(H, N, 1, device=dev, stream=stream)
        # thresholds: Eq. 3 on the post-gate activations of 256 calibration vectors
        xc = torch.from_numpy(inputs.activations_bf16(N_CALIB, H, seed=inputs.SEED_CALIB).view(np.int16)).to(dev)
        a = torch.empty(N_CALIB, N, dtype=torch.float32, device=dev)
        sats.gate_act(layers[0], xc, a, stream=stream)
        sel = torch.empty(sats.select_workspace_bytes(), dtype=torch.uint8, device=dev)
        ts = [sats.percentile_threshold(a, s, sel, stream=stream) for s in SPARSITY]
        del a, xc
        x = torch.from_numpy(inputs.activations_bf16(1, H).view(np.int16)).to(dev)
        y = torch.empty(1, H, dtype=torch.float32, device=dev)
        idx = torch.empty(1, N, dtype=torch.int32, device=dev)
        cnt = torch.empty(1, dtype=torch.int32, device=dev)
    stream.synchronize()

    if args.profile_batch:
        # small capture case for ncu: one layer copy, `steps` calls at one batch size
        B = args.profile_batch
        xb = torch.randn(B, H, device=dev, dtype=torch.float32).to(torch.bfloat16).view(torch.int16)
        yb = torch.empty(B, H, dtype=torch.float32, device=dev)
        wsb = sats.Workspace(H, N, B, device=dev, stream=stream)
        for i in range(max(args.warmup, 1) + args.steps):
            sats.sparse_mlp(layers[0], xb, ts[0], yb, wsb, stream=stream)
        stream.synchronize()
        ok = sats.get_error(wsb, stream=stream) == sats.OK
        if rank == 0:
            print(json.dumps({"profile_case": "llama_layer_4096x14336_b%d" % B, "calls": max(args.warmup, 1) + args.steps,
                              "tensor_cores": sats.uses_tensor_cores(H, B), "status_ok": ok}))
        for l in layers:
            l.close()
        if not ok:
            raise RuntimeError("device status after the profile calls")
        return

    calls = [(i, ts[i]) for i in range(len(SPARSITY))]
    copy = [0]

    def one_call(si, t, ev0=None, ev1=None):
        layer = layers[copy[0] % len(layers)]
        copy[0] += 1
        if ev0 is not None:
            ev0.record(stream)
        sats.sparse_mlp(layer, x, t, y, ws, idx, cnt, stream=stream)
        if ev1 is not None:
            ev1.record(stream)

    # realised sparsity per level
    realised = []
    for si, t in calls:
        one_call(si, t)
        stream.synchronize()
        realised.append(1.0 - int(cnt.item()) / N)
    assert sats.get_error(ws, stream=stream) == sats.OK

    for _ in range(max(args.warmup, 3)):
        for si, t in calls:
            one_call(si, t)
    K = args.steps
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks = Clocks(local)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    clocks.start()
    time.sleep(0.3)
    # timed region: K steps, each the three calls back to back (launches overlap
    # their prologue with the previous call's tail)
    start.record(stream)
    for k in range(K):
        for si, t in calls:
            one_call(si, t)
    stop.record(stream)
    stop.synchronize()
    # average launch duration per sparsity level: K launches of that level back
    # to back on the same stream, bracketed by events
    mean_us = []
    for si, t in calls:
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for k in range(K):
            one_call(si, t)
        e1.record(stream)
        e1.synchronize()
        mean_us.append(1e3 * e0.elapsed_time(e1) / K)
    # the same without index lists (y only), outside the timed region: what the lists cost
    nolist_us = []
    if not args.profile:
        for si, t in calls:
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for k in range(K):
                layer = layers[copy[0] % len(layers)]
                copy[0] += 1
                sats.sparse_mlp(layer, x, t, y, ws, stream=stream)
            e1.record(stream)
            e1.synchronize()
            nolist_us.append(1e3 * e0.elapsed_time(e1) / K)
    torch.cuda.synchronize(dev)
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    status = sats.get_error(ws, stream=stream)
    if status != sats.OK:
        raise RuntimeError("device status after the timed region: " + sats.status_string(status))
    total_ms = start.elapsed_time(stop)

    if args.profile:
        if rank == 0:
            print(json.dumps({"profile_case": WORKLOAD, "per_call_us": mean_us, "realised": realised}))
        for l in layers:
            l.close()
        return

    # dense path on the same copies, for the speedup
    for i in range(3):
        sats.dense_mlp(layers[i % len(layers)], x, y, ws, stream=stream)
    d0, d1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    d0.record(stream)
    for i in range(K):
        sats.dense_mlp(layers[i % len(layers)], x, y, ws, stream=stream)
    d1.record(stream)
    d1.synchronize()
    dense_us = 1e3 * d0.elapsed_time(d1) / K

    # batched decode and prefill on the tensor-core path (50 % threshold), same rotating copies
    batched = {}
    if not args.no_batched:
        bf16_peak, bf16_kind = _bf16_peak()
        for B in BATCHES:
            xb = torch.randn(B, H, device=dev, dtype=torch.float32).to(torch.bfloat16).view(torch.int16)
            yb = torch.empty(B, H, dtype=torch.float32, device=dev)
            wsb = sats.Workspace(H, N, B, device=dev, stream=stream)
            Kb = max(4, min(K, int(4e4 / (60 + 0.33 * B))))
            for i in range(3):
                sats.sparse_mlp(layers[i % len(layers)], xb, ts[0], yb, wsb, stream=stream)
            b0, b1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            b0.record(stream)
            for i in range(Kb):
                sats.sparse_mlp(layers[i % len(layers)], xb, ts[0], yb, wsb, stream=stream)
            b1.record(stream)
            b1.synchronize()
            if sats.get_error(wsb, stream=stream) != sats.OK:
                raise RuntimeError("device status after the batched calls")
            us = 1e3 * b0.elapsed_time(b1) / Kb
            wbytes = 6.0 * H * N + B * H * 2.0 + B * H * 4.0
            flops = 6.0 * B * H * N
            batched[str(B)] = {"us_per_call": us, "tokens_per_s": B / (us * 1e-6),
                               "hbm_gbs": wbytes / (us * 1e-6) / 1e9, "tflops": flops / (us * 1e-6) / 1e12,
                               "tensor_frac_of_%s" % bf16_kind: flops / (us * 1e-6) / 1e12 / bf16_peak,
                               "calls": Kb, "path": "tensor cores" if sats.uses_tensor_cores(H, B) else "fused"}
            del xb, yb, wsb

    # end to end through the C ABI with host buffers: each step copies its tokens' x (one per
    # call) host->device at once, runs the calls back to back (chained by programmatic dependent
    # launch) and reads every y and count back at once, then waits for them on the host
    nc = len(calls)
    xh = torch.from_numpy(np.repeat(inputs.activations_bf16(1, H), nc, axis=0).view(np.int16)).pin_memory()
    yh = torch.empty(nc, H, dtype=torch.float32).pin_memory()
    ch = torch.empty(nc, dtype=torch.int32).pin_memory()
    xe = torch.empty(nc, H, dtype=torch.int16, device=dev)
    ye = torch.empty(nc, H, dtype=torch.float32, device=dev)
    ce = torch.empty(nc, dtype=torch.int32, device=dev)
    Ke = max(10, K // 4)
    e2e_s, e2e_e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    for rep in range(2):
        if rep == 1:
            e2e_s.record(stream)
        for k in range(Ke if rep else 3):
            with torch.cuda.stream(stream):
                xe.copy_(xh, non_blocking=True)
            for si, t in calls:
                layer = layers[copy[0] % len(layers)]
                copy[0] += 1
                sats.sparse_mlp(layer, xe[si:si + 1], t, ye[si:si + 1], ws, idx, ce[si:si + 1], stream=stream)
            with torch.cuda.stream(stream):
                yh.copy_(ye, non_blocking=True)
                ch.copy_(ce, non_blocking=True)
            stream.synchronize()
        if rep == 1:
            e2e_e.record(stream)
    stream.synchronize()
    e2e_us = 1e3 * e2e_s.elapsed_time(e2e_e) / (Ke * nc)

    # the same step as a serving loop replays it: captured once in a CUDA graph (the host->device
    # copy from pinned memory, the calls on three layer copies, the device->host copies), replayed
    # and waited for on the host every step (reported beside e2e, not in its place)
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        xe.copy_(xh, non_blocking=True)
        for si, t in calls:
            sats.sparse_mlp(layers[si % len(layers)], xe[si:si + 1], t, ye[si:si + 1], ws, idx, ce[si:si + 1],
                            stream=stream)
        yh.copy_(ye, non_blocking=True)
        ch.copy_(ce, non_blocking=True)
    g0, g1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):   # a replay runs on the current stream
        for _ in range(3):
            graph.replay()
            stream.synchronize()
        g0.record(stream)
        for _ in range(Ke):
            graph.replay()
            stream.synchronize()
        g1.record(stream)
    stream.synchronize()
    e2e_graph_us = 1e3 * g0.elapsed_time(g1) / (Ke * nc)
    del graph

    # the other four workloads at their full sizes, compact (one GPU; not part of the headline value)
    configs = {}
    if not args.no_configs and world == 1:
        for l in layers:
            l.close()
        layers = []
        hbm_peak, peak_kind = _peaks()
        bf16_peak, bf16_kind = _bf16_peak()
        t_cfg = time.perf_counter()
        clk_cfg = Clocks(local)
        clk_cfg.start()
        with torch.cuda.stream(stream):
            configs["small_layer_512x1408_b1"] = _wl_small_layer(sats, dev, stream, 200)
            configs["llama_stack_32x4096x14336_b1x128"] = _wl_llama_stack(sats, dev, stream, 128, hbm_peak,
                                                                          peak_kind)
            torch.cuda.empty_cache()
            configs["qwen_stack_36x4096x12288_routed"] = _wl_qwen_stack(sats, dev, stream, [1, 8, 32, 64], 10)
            torch.cuda.empty_cache()
            configs["llama_layer_prefill_routed"] = _wl_prefill(sats, dev, stream, [0.4, 0.9], [256, 2048], 10,
                                                                bf16_peak, bf16_kind)
        configs["clocks"] = clk_cfg.stop()
        configs["seconds"] = time.perf_counter() - t_cfg

    # aggregate over ranks (replicas): max time
    total_ms, e2e_us = _max_over_ranks([total_ms, e2e_us], world, device=dev)
    if rank == 0:
        hbm_peak, peak_kind = _peaks()
        per = {}
        bytes_all, us_all = 0.0, 0.0
        for i, s in enumerate(SPARSITY):
            kept = (1.0 - realised[i]) * N
            algo = 2.0 * H * N + kept * 4.0 * H + 2.0 * H + 4.0 * H + 4.0 * kept + 4.0
            gbs = algo / (mean_us[i] * 1e-6) / 1e9
            per[str(s)] = {"us": mean_us[i], "realised_sparsity": realised[i], "algo_bytes": algo,
                           "achieved_gbs": gbs, "frac_of_%s" % peak_kind: gbs / hbm_peak,
                           "frac_of_8tbs": gbs / NOMINAL_HBM_GBS, "speedup_vs_dense": dense_us / mean_us[i]}
            if nolist_us:
                per[str(s)]["us_without_index_lists"] = nolist_us[i]
            bytes_all += algo
            us_all += mean_us[i]
        achieved = bytes_all / (us_all * 1e-6) / 1e9
        traffic = _ncu_traffic()
        value = _us_per_token(total_ms, K, len(calls), world)
        line = {
            "metric": METRIC, "value": value, "unit": "us/token", "n_gpus": world, "steps": K,
            "warmup": max(args.warmup, 3), "ms_per_step": total_ms / K, "higher_is_better": False,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": _headline_config(world),
            "per_sparsity": per,
            "dense": {"us": dense_us},
            "batched": batched,
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": hbm_peak, "unit": "GB/s",
                         "frac": achieved / hbm_peak, "peak_kind": peak_kind,
                         "traffic": None if traffic is None else
                         sum(traffic[s] for s in SPARSITY) / len(SPARSITY),
                         "kernel": "fused_mlp_kernel<1,2,0>"},
            "e2e": {"value": e2e_us, "unit": "us/token", "h2d_bytes_per_step": len(calls) * 2 * H,
                    "d2h_bytes_per_step": len(calls) * (4 * H + 4),
                    "graph_replayed_step_us_per_token": e2e_graph_us},
            "gpu_launches": K * len(calls),
            "clocks": clk,
        }
        if configs:
            line["configs"] = configs
        if not args.no_cpu_baseline:
            orc, w_or, ts_or = _oracle_setup()
            us, sample = _oracle_one_core(orc, w_or, ts_or, args.cpu_seconds)
            line["cpu_baseline"] = {"value": us, "unit": "us/token", "cores": 1, "kind": "oracle", "sample": sample}
            threads = _host_threads()
            us_all, _ = _oracle_all_cores(orc, w_or, ts_or, 2, threads)
            line["cpu_baseline_all_cores"] = {
                "value": us_all, "unit": "us/token", "cores": threads, "os_cpu_count": os.cpu_count(),
                "kind": "oracle", "sample": "%d single-token calls, %d at a time (one per host core)"
                                            % (2 * threads, threads)}
        print(json.dumps(line))
    for l in layers:
        l.close()
    if world > 1:
        dist.destroy_process_group()


# ---------------------------------------------------------------------------- other workloads
def _eq3_stack_thresholds(sats, layers, nws, targets, eps, xc, stream):
    """Per-block thresholds for the bench (setup, not timed, not a parity input): the Eq. 3
    percentile of the post-gate magnitudes of fp32 calibration vectors carried through the
    earlier, already thresholded blocks, computed with the library's own RMSNorm, gate and
    percentile kernels."""
    import torch
    C, H = xc.shape
    N = layers[0].N
    x = xc.clone()
    n = torch.empty_like(x)
    a = torch.empty(C, N, dtype=torch.float32, device=x.device)
    sel = torch.empty(sats.select_workspace_bytes(), dtype=torch.uint8, device=x.device)
    ws = sats.Workspace(H, N, C, device=x.device, stream=stream)
    ts = []
    for l, layer in enumerate(layers):
        sats.rmsnorm(x, nws[l], eps, n, stream=stream)
        sats.gate_act_f32(layer, n, a, stream=stream)
        t = sats.percentile_threshold(a, float(targets[l]), sel, stream=stream)
        ts.append(t)
        sats.mlp_stack([layer], [nws[l]], [t], eps, x, ws, stream=stream)
    stream.synchronize()
    return ts


def _timed(stream, fn, reps):
    import torch
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(reps):
        fn(i)
    e1.record(stream)
    e1.synchronize()
    return 1e3 * e0.elapsed_time(e1) / reps


def _graph_timed(stream, fn, n_calls, reps):
    """Device time per call of `n_calls` calls captured once into a CUDA graph and replayed
    `reps` times back to back (for calls shorter than the host's launch time)."""
    import torch
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for i in range(n_calls):
            fn(i)
    stream.synchronize()
    with torch.cuda.stream(stream):
        g.replay()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            g.replay()
        e1.record(stream)
    e1.synchronize()
    return 1e3 * e0.elapsed_time(e1) / (reps * n_calls)


def _wl_small_layer(sats, dev, stream, steps):
    """Hidden 512 / intermediate 1408, one decode token, t at the 50th percentile of 64 calibration
    vectors; 64 rotating copies of the layer (184 MB, weights from HBM) and one copy (L2-resident)."""
    import torch
    spec = inputs.WORKLOADS["small_layer_512x1408_b1"]
    H, N = spec["H"], spec["N"]
    layers = [sats.Layer(*inputs.mlp_weights_device(H, N, layer=l), stream=stream) for l in range(64)]
    ws = sats.Workspace(H, N, 1, device=dev, stream=stream)
    xc = torch.from_numpy(inputs.activations_bf16(spec["calib"], H, seed=inputs.SEED_CALIB).view(np.int16)).to(dev)
    a = torch.empty(spec["calib"], N, dtype=torch.float32, device=dev)
    sats.gate_act(layers[0], xc, a, stream=stream)
    sel = torch.empty(sats.select_workspace_bytes(), dtype=torch.uint8, device=dev)
    t = sats.percentile_threshold(a, 0.5, sel, stream=stream)
    x = torch.from_numpy(inputs.activations_bf16(1, H).view(np.int16)).to(dev)
    y = torch.empty(1, H, dtype=torch.float32, device=dev)
    idx = torch.empty(1, N, dtype=torch.int32, device=dev)
    cnt = torch.empty(1, dtype=torch.int32, device=dev)
    call = lambda i: sats.sparse_mlp(layers[i % 64], x, t, y, ws, idx, cnt, stream=stream)
    for i in range(64):
        call(i)
    stream.synchronize()
    kept = int(cnt.item())
    # a call of this layer is shorter than the host's launch time: the device time comes from
    # 64 calls (one per copy) captured in a CUDA graph and replayed; the eagerly launched loop
    # is reported beside it
    us_cold = _graph_timed(stream, call, 64, max(4, steps // 64))
    us_hot = _graph_timed(stream, lambda i: call(0), 64, max(4, steps // 64))
    us_eager = _timed(stream, call, steps)
    if sats.get_error(ws, stream=stream) != sats.OK:
        raise RuntimeError("device status after the small-layer calls")
    for l in layers:
        l.close()
    algo = 2.0 * H * N + 4.0 * H * kept + 2.0 * H + 4.0 * H + 4.0 * kept + 4.0
    return {"us_per_token": us_cold, "us_l2_resident": us_hot, "us_per_token_eager_launches": us_eager,
            "timing": "64 calls (64 rotating layer copies, 184 MB) in a CUDA graph, replayed back to back",
            "realised_sparsity": 1.0 - kept / N, "algo_bytes": algo, "achieved_gbs": algo / us_cold / 1e3,
            "calls": 64 * max(4, steps // 64)}


def _wl_llama_stack(sats, dev, stream, tokens, hbm_peak, hbm_kind):
    """32 Llama-3.1-8B-shaped blocks (RMSNorm -> MLP -> residual), `tokens` decode tokens one per
    call, per-block targets evenly spread over [55 %, 85 %] (mean 70 %)."""
    import torch
    spec = inputs.WORKLOADS["llama_stack_32x4096x14336_b1x128"]
    H, N, L, eps = spec["H"], spec["N"], spec["L"], spec["eps"]
    targets = list(inputs.stack_sparsity_targets(L, *spec["sparsity_range"]))
    layers = [sats.Layer(*inputs.mlp_weights_device(H, N, layer=l), stream=stream) for l in range(L)]
    nws = [torch.from_numpy(inputs.norm_weight(H, layer=l)).to(dev) for l in range(L)]
    xc = torch.from_numpy(inputs.activations_f32(64, H, seed=inputs.SEED_CALIB)).to(dev)
    ts = _eq3_stack_thresholds(sats, layers, nws, targets, eps, xc, stream)
    x0 = torch.from_numpy(inputs.activations_f32(tokens, H, seed=inputs.SEED_X + 3)).to(dev)
    ws = sats.Workspace(H, N, 1, device=dev, stream=stream)
    trace = torch.empty((L, 1, N), dtype=torch.uint8, device=dev)
    kept_sum = torch.zeros(L, dtype=torch.float64, device=dev)
    x = x0.clone()
    for tok in range(tokens):      # keep masks of every token (untimed), for the realised sparsity
        sats.mlp_stack(layers, nws, ts, eps, x[tok:tok + 1], ws, keep_trace=trace, stream=stream)
        with torch.cuda.stream(stream):
            kept_sum += trace[:, 0].sum(dim=1).double()
    stream.synchronize()
    kept = (kept_sum / tokens).cpu().numpy()          # [L] mean kept neurons per token
    del trace
    x = x0.clone()
    step = lambda i: sats.mlp_stack(layers, nws, ts, eps, x[i % tokens:i % tokens + 1], ws, stream=stream)
    for i in range(3):
        step(i)
    x.copy_(x0)
    us = _timed(stream, step, tokens)      # every token once through the stack
    if sats.get_error(ws, stream=stream) != sats.OK:
        raise RuntimeError("device status after the stack calls")
    for l in layers:
        l.close()
    algo = float(sum(2.0 * H * N + 4.0 * H * k + 12.0 * H for k in kept))
    return {"us_per_token": us, "tokens_per_s": 1e6 / us, "tokens": tokens,
            "realised_sparsity_mean": float(1.0 - kept.mean() / N),
            "realised_sparsity_range": [float(1.0 - kept.max() / N), float(1.0 - kept.min() / N)],
            "algo_bytes_per_token": algo, "achieved_gbs": algo / us / 1e3,
            "frac_of_%s" % hbm_kind: algo / us / 1e3 / hbm_peak}


def _wl_qwen_stack(sats, dev, stream, batches, reps_max):
    """36 Qwen3-8B-shaped blocks with routing over a 151936-entry table (30 % dense), decode
    batches of uniform token ids, sparse path at 50 % per block."""
    import torch
    spec = inputs.WORKLOADS["qwen_stack_36x4096x12288_routed"]
    H, N, L, V, eps = spec["H"], spec["N"], spec["L"], spec["V"], spec["eps"]
    layers = [sats.Layer(*inputs.mlp_weights_device(H, N, layer=l, seed=inputs.SEED_WEIGHTS + 100), stream=stream)
              for l in range(L)]
    nws = [torch.from_numpy(inputs.norm_weight(H, layer=l)).to(dev) for l in range(L)]
    xc = torch.from_numpy(inputs.activations_f32(64, H, seed=inputs.SEED_CALIB)).to(dev)
    ts = _eq3_stack_thresholds(sats, layers, nws, [spec["sparsity"]] * L, eps, xc, stream)
    lut = torch.from_numpy(inputs.routing_lut(V, spec["p_dense"])).to(dev)
    res = {}
    for B in batches:
        x0 = torch.from_numpy(inputs.activations_f32(B, H, seed=inputs.SEED_X + 40 + B)).to(dev)
        ids = torch.from_numpy(inputs.token_ids_uniform(B, V, seed=inputs.SEED_IDS + B)).to(dev)
        ws = sats.Workspace(H, N, B, device=dev, stream=stream)
        reps = reps_max
        xs = x0.repeat(reps + 3, 1, 1)        # a fresh copy of the batch per step
        step = lambda i: sats.mlp_stack(layers, nws, ts, eps, xs[i], ws, token_ids=ids, lut=lut, stream=stream)
        for i in range(3):
            step(reps + i)
        us = _timed(stream, step, reps)
        if sats.get_error(ws, stream=stream) != sats.OK:
            raise RuntimeError("device status after the routed stack calls")
        res[str(B)] = {"us_per_step": us, "tokens_per_s": B / (us * 1e-6),
                       "dense_tokens": int(lut[ids.long()].sum()),
                       "path": "tensor cores" if sats.uses_tensor_cores(H, B) else "fused",
                       "weight_gbs_if_all_weights_read": L * 6.0 * H * N / us / 1e3}
        del xs, ws
    for l in layers:
        l.close()
    return res


def _wl_prefill(sats, dev, stream, sparsities, batches, reps_max, bf16_peak, bf16_kind):
    """One Llama-shaped block with routing (20 % of a 128256-entry table dense, Zipf(1.1) ids) at
    prefill sizes; dense-equivalent and method-work (algorithmic) FLOP rates."""
    import torch
    spec = inputs.WORKLOADS["llama_layer_prefill_routed"]
    H, N, V = inputs.LLAMA_H, inputs.LLAMA_N, spec["V"]
    eps = 1e-5
    layers = [sats.Layer(*inputs.mlp_weights_device(H, N, layer=l, seed=inputs.SEED_WEIGHTS + 200), stream=stream)
              for l in range(2)]
    nw = torch.from_numpy(inputs.norm_weight(H)).to(dev)
    lut = torch.from_numpy(inputs.routing_lut(V, spec["p_dense"], seed=inputs.SEED_LUT + 5)).to(dev)
    xc = torch.from_numpy(inputs.activations_f32(256, H, seed=inputs.SEED_CALIB)).to(dev)
    res = {}
    for k in sparsities:
        t = _eq3_stack_thresholds(sats, layers[:1], [nw], [k], eps, xc, stream)[0]
        for B in batches:
            ids = torch.from_numpy(inputs.token_ids_zipf(B, V, seed=inputs.SEED_IDS + B)).to(dev)
            x0 = torch.from_numpy(inputs.activations_f32(B, H, seed=inputs.SEED_X + 50 + B)).to(dev)
            ws = sats.Workspace(H, N, B, device=dev, stream=stream)
            dense = lut[ids.long()].bool()
            trace = torch.empty((1, B, N), dtype=torch.uint8, device=dev)
            xt = x0.clone()
            sats.mlp_stack([layers[0]], [nw], [t], eps, xt, ws, token_ids=ids, lut=lut, keep_trace=trace,
                           stream=stream)
            kept_sparse = float(trace[0][~dense].double().mean()) if bool((~dense).any()) else 0.0
            nd = int(dense.sum())
            del trace, xt
            reps = max(4, min(reps_max, int(2e4 / B)))
            xs = x0.repeat(reps + 3, 1, 1)
            step = lambda i: sats.mlp_stack([layers[i % 2]], [nw], [t], eps, xs[i], ws, token_ids=ids, lut=lut,
                                            stream=stream)
            for i in range(3):
                step(reps + i)
            us = _timed(stream, step, reps)
            if sats.get_error(ws, stream=stream) != sats.OK:
                raise RuntimeError("device status after the prefill calls")
            flops = 6.0 * B * H * N
            method = nd * 6.0 * H * N + (B - nd) * (2.0 + 4.0 * kept_sparse) * H * N
            res["%s@%d" % (k, B)] = {"us_per_call": us, "tokens_per_s": B / (us * 1e-6),
                                     "tflops_dense_equivalent": flops / us / 1e6,
                                     "tensor_frac_of_%s" % bf16_kind: flops / us / 1e6 / bf16_peak,
                                     "method_tflops": method / us / 1e6,
                                     "method_frac_of_%s" % bf16_kind: method / us / 1e6 / bf16_peak,
                                     "dense_fraction_of_tokens": nd / B,
                                     "sparse_tokens_realised_sparsity": 1.0 - kept_sparse}
            del xs, ws
    for l in layers:
        l.close()
    return res


def run_workload(args):
    """The other four workloads (one JSON line each; not the headline)."""
    import torch

    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_08991_gb300 import sats

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    stream = torch.cuda.Stream(device=dev)
    hbm_peak, hbm_kind = _peaks()
    bf16_peak, bf16_kind = _bf16_peak()
    wl = args.workload
    spec = inputs.WORKLOADS[wl]
    out = {"workload": wl, "data": "synthetic", "hbm_peak_gbs": hbm_peak, "bf16_peak_tflops": bf16_peak,
           "peak_kind": hbm_kind}
    clocks = Clocks(0)
    with torch.cuda.stream(stream):
        if wl == "small_layer_512x1408_b1":
            clocks.start()
            r = _wl_small_layer(sats, dev, stream, args.steps)
            clk = clocks.stop()
            out.update({"metric": "us/token (one layer)", "value": r["us_per_token"], "unit": "us/token",
                        "clocks": clk, **r})
        elif wl == "llama_stack_32x4096x14336_b1x128":
            clocks.start()
            r = _wl_llama_stack(sats, dev, stream, spec["tokens"], hbm_peak, hbm_kind)
            clk = clocks.stop()
            out.update({"metric": "us/token through the %d-block stack (decode, one token per call)" % spec["L"],
                        "value": r["us_per_token"], "unit": "us/token", "clocks": clk, **r})
        elif wl == "qwen_stack_36x4096x12288_routed":
            clocks.start()
            res = _wl_qwen_stack(sats, dev, stream, spec["batches"], max(10, args.steps // 4))
            clk = clocks.stop()
            out.update({"metric": "us per decode step through the %d-block routed stack" % spec["L"],
                        "value": res[str(spec["batches"][-1])]["us_per_step"], "unit": "us/step",
                        "per_batch": res, "clocks": clk})
        elif wl == "llama_layer_prefill_routed":
            clocks.start()
            res = _wl_prefill(sats, dev, stream, spec["sparsity"], spec["batches"], args.steps, bf16_peak, bf16_kind)
            clk = clocks.stop()
            out.update({"metric": "us per prefill call (one routed block)", "value": res["0.6@2048"]["us_per_call"],
                        "unit": "us/call", "per_case": res, "clocks": clk})
        elif wl == "union_batch_llama_4096x14336":
            # the union path (sats_sparse_mlp_union) against the default batched path on
            # the same calls: independent tokens (rho = 0) and strongly correlated ones
            H, N = spec["H"], spec["N"]
            layers = [sats.Layer(*inputs.mlp_weights_device(H, N, layer=l)) for l in range(LAYER_COPIES)]
            xc = torch.from_numpy(inputs.activations_bf16(spec["calib"], H, seed=inputs.SEED_CALIB).view(np.int16)).to(dev)
            a = torch.empty(spec["calib"], N, dtype=torch.float32, device=dev)
            sats.gate_act(layers[0], xc, a, stream=stream)
            sel = torch.empty(sats.select_workspace_bytes(), dtype=torch.uint8, device=dev)
            ts = {k: sats.percentile_threshold(a, k, sel, stream=stream) for k in spec["sparsity"]}
            del a
            res = {}
            clocks.start()
            for rho in spec["rho"]:
                for B in spec["batches"]:
                    ws = sats.Workspace(H, N, B, device=dev)
                    xb = (inputs.activations_bf16(B, H, seed=inputs.SEED_X + B) if rho == 0.0 else
                          inputs.activations_correlated_bf16(B, H, rho, seed=inputs.SEED_X + B))
                    x = torch.from_numpy(xb.view(np.int16)).to(dev)
                    y = torch.empty(B, H, dtype=torch.float32, device=dev)
                    idx = torch.empty(B, N, dtype=torch.int32, device=dev)
                    cnt = torch.empty(B, dtype=torch.int32, device=dev)
                    for k, t in ts.items():
                        sats.sparse_mlp_union(layers[0], x, t, y, ws, idx, cnt, stream=stream)
                        stream.synchronize()
                        c = cnt.cpu().numpy()
                        keep = np.zeros((B, N), bool)
                        ii = idx.cpu().numpy()
                        for m in range(B):
                            keep[m, ii[m, :c[m]]] = True
                        U = int(keep.any(axis=0).sum())
                        runs = {}
                        for name, fn in (("union", sats.sparse_mlp_union), ("default", sats.sparse_mlp)):
                            call = lambda i, fn=fn: fn(layers[i % LAYER_COPIES], x, t, y, ws, stream=stream)
                            for i in range(args.warmup + 3):
                                call(i)
                            runs[name] = _timed(stream, call, max(args.steps // 4, 20))
                        algo_union = 2.0 * H * N + 4.0 * H * U + 2.0 * B * H + 4.0 * B * H
                        res["rho%.1f_B%d_s%.1f" % (rho, B, k)] = {
                            "union_fraction": U / N, "mean_sparsity": 1.0 - float(c.mean()) / N,
                            "us_union": runs["union"], "us_default": runs["default"],
                            "union_bytes": algo_union, "union_gbs": algo_union / runs["union"] / 1e3,
                            "default_gbs_all_weights": 6.0 * H * N / runs["default"] / 1e3}
                    del ws
            clk = clocks.stop()
            out.update({"metric": "us per call, union path vs default batched path", "unit": "us/call",
                        "value": min(v["us_union"] for v in res.values()), "per_case": res,
                        "input": "x ~ N(0,1) per token (rho 0) or rho z_0 + sqrt(1-rho^2) z_m (rho 0.9), bf16",
                        "clocks": clk})
        elif wl == "lora_llama_layer_4096x14336_b1":
            # sats_sparse_mlp_lora against sats_sparse_mlp on the same layer copies and thresholds
            H, N = spec["H"], spec["N"]
            layers = [sats.Layer(*inputs.mlp_weights_device(H, N, layer=l)) for l in range(LAYER_COPIES)]
            xc = torch.from_numpy(inputs.activations_bf16(spec["calib"], H, seed=inputs.SEED_CALIB).view(np.int16)).to(dev)
            a = torch.empty(spec["calib"], N, dtype=torch.float32, device=dev)
            sats.gate_act(layers[0], xc, a, stream=stream)
            sel = torch.empty(sats.select_workspace_bytes(), dtype=torch.uint8, device=dev)
            ts = {k: sats.percentile_threshold(a, k, sel, stream=stream) for k in spec["sparsity"]}
            del a
            ws = sats.Workspace(H, N, 1, device=dev)
            x = torch.from_numpy(inputs.activations_bf16(1, H).view(np.int16)).to(dev)
            y = torch.empty(1, H, dtype=torch.float32, device=dev)
            idx = torch.empty(1, N, dtype=torch.int32, device=dev)
            cnt = torch.empty(1, dtype=torch.int32, device=dev)
            reps = max(args.steps, 50)
            res = {}
            clocks.start()
            for k, t in ts.items():
                base = lambda i, t=t: sats.sparse_mlp(layers[i % LAYER_COPIES], x, t, y, ws, idx, cnt, stream=stream)
                for i in range(args.warmup + 3):
                    base(i)
                res["base_s%.1f" % k] = {"us": _timed(stream, base, reps)}
            for r in spec["ranks"]:
                los = [sats.Lora(layers[l], *(torch.from_numpy(m.view(np.int16)).to(dev)
                                              for m in inputs.lora_adapter(H, N, r, seed=7000 + l)),
                                 scale=spec["scale"], stream=stream) for l in range(LAYER_COPIES)]
                for k, t in ts.items():
                    call = lambda i, t=t: sats.sparse_mlp_lora(layers[i % LAYER_COPIES], los[i % LAYER_COPIES], x, t, y,
                                                               ws, idx, cnt, stream=stream)
                    for i in range(args.warmup + 3):
                        call(i)
                    stream.synchronize()
                    kept = int(cnt.item())
                    us = _timed(stream, call, reps)
                    base_bytes = 2.0 * H * N + 4.0 * H * kept + 2.0 * H + 4.0 * H + 4.0 * kept + 4.0
                    lora_bytes = N * 6.0 * r + H * 4.0 * r + r * 2.0 * H   # adapter blocks, A_gate | A_up, B_down
                    res["r%d_s%.1f" % (r, k)] = {
                        "us": us, "overhead_us": us - res["base_s%.1f" % k]["us"], "realised_sparsity": 1.0 - kept / N,
                        "algo_bytes": base_bytes + lora_bytes, "achieved_gbs": (base_bytes + lora_bytes) / us / 1e3}
                for l in los:
                    l.close()
            clk = clocks.stop()
            out.update({"metric": "us/token, LoRA-aware sparse MLP (one layer)", "unit": "us/token",
                        "value": res["r16_s0.5"]["us"], "per_case": res, "clocks": clk,
                        "adapter": "synthetic rank-r factors N(0, 0.02) in bf16 on gate, up and down, scale 1"})
        elif wl == "sats_calibration_llama_32x4096x14336":
            H, N, L, C = spec["H"], spec["N"], spec["L"], spec["calib"]
            layers = [sats.Layer(*inputs.mlp_weights_device(H, N, layer=l)) for l in range(L)]
            nws = [torch.from_numpy(inputs.norm_weight(H, layer=l)).to(dev) for l in range(L)]
            xc = torch.from_numpy(inputs.activations_f32(C, H, seed=inputs.SEED_CALIB)).to(dev)
            torch.cuda.synchronize()
            # one Eq. 6 evaluation for its cost per candidate
            n0 = torch.empty_like(xc)
            sats.rmsnorm(xc, nws[0], spec["eps"], n0, stream=stream)
            sats.layer_err(layers[0], n0, [0.1], stream=stream)
            t0 = time.perf_counter()
            sats.layer_err(layers[0], n0, [0.05 * k for k in range(1, 9)], stream=stream)
            per_cand = (time.perf_counter() - t0) / 8
            clocks.start()
            t0 = time.perf_counter()
            r = sats.sats_calibrate(layers, nws, spec["eps"], xc, spec["target"], K0=spec["K0"], K1=spec["K1"],
                                    guardrail=True, stream=stream)
            el = time.perf_counter() - t0
            clk = clocks.stop()
            out.update({"metric": "seconds for the SATS calibration of the %d-block stack" % L, "value": el,
                        "unit": "s", "calibration_vectors": C, "coarse_candidates": spec["K0"] - 1,
                        "fine_candidates": spec["K1"], "eq6_evaluations": L * (spec["K0"] - 1 + spec["K1"]) + 1,
                        "seconds_per_eq6_candidate_one_block": per_cand, "target_sparsity": spec["target"],
                        "realised_S": r["S"], "budget": r["b"], "thresholds": [round(v, 5) for v in r["t"]],
                        "clocks": clk})
        elif wl == "route_calibration_qwen_v151936":
            V = spec["V"]
            ids, lb, ls = inputs.routing_corpus(spec["corpus"], V)
            held = inputs.token_ids_zipf(spec["heldout"], V, seed=inputs.SEED_IDS + 200)
            ids_d, lb_d, ls_d = (torch.from_numpy(a).to(dev) for a in (ids, lb, ls))
            held_d = torch.from_numpy(held).to(dev)
            sats.token_scores(ids_d, lb_d, ls_d, V, stream=stream)      # warm-up
            clocks.start()
            t0 = time.perf_counter()
            score = sats.token_scores(ids_d, lb_d, ls_d, V, stream=stream)
            t_scores = time.perf_counter() - t0
            res = {}
            for r_tar in spec["targets"]:
                t0 = time.perf_counter()
                tau, R, lut = sats.route_calibrate(score, held_d, r_tar, stream=stream)
                res[str(r_tar)] = {"tau": tau, "R": R, "seconds": time.perf_counter() - t0,
                                   "dense_fraction_of_vocab": float(lut.float().mean())}
            clk = clocks.stop()
            out.update({"metric": "seconds for the token scores of the routing corpus (Eqs. 11-12)",
                        "value": t_scores, "unit": "s", "corpus_occurrences": spec["corpus"],
                        "heldout_occurrences": spec["heldout"], "occurrences_per_s": spec["corpus"] / t_scores,
                        "per_target": res, "clocks": clk})
        else:
            raise SystemExit("unknown workload " + wl)
    print(json.dumps(out))


PROFILE_CASES = ("route", "batch64", "union", "lora", "small", "stack", "prefill")


def run_profile_case(args):
    """Small capture cases for ncu, one kernel group each, `warmup + steps` launches of it:
    route (the routing kernel at 64 and 2048 tokens over the Qwen-shaped vocabulary),
    batch64 (the Llama-shaped layer at 64 tokens with index lists: the skinny tensor-core pair
    and the kept-list kernel), union (the union path at 8 tokens, 90 %), lora (the LoRA-aware
    decode kernel at rank 16, one token, 70 %), small (the small-layer cluster kernel), stack
    (one Llama-shaped block of a routed stack at 64 tokens: the RMSNorm/split kernel with the
    routing gather, then the skinny pair) and prefill (the same block at 2048 tokens, 90 %: the
    split kernel, then the prefill pair with fp32 activations).  Prints one JSON line."""
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_08991_gb300 import sats
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(0)
    stream = torch.cuda.Stream(device=dev)
    n_calls = max(args.warmup, 1) + args.steps
    case = args.profile_case

    def threshold(layer, H, N, k, n_cal=64):
        xc = torch.from_numpy(inputs.activations_bf16(n_cal, H, seed=inputs.SEED_CALIB).view(np.int16)).to(dev)
        a = torch.empty(n_cal, N, dtype=torch.float32, device=dev)
        sats.gate_act(layer, xc, a, stream=stream)
        sel = torch.empty(sats.select_workspace_bytes(), dtype=torch.uint8, device=dev)
        return sats.percentile_threshold(a, k, sel, stream=stream)

    info = {"profile_case": case, "calls": n_calls}
    with torch.cuda.stream(stream):
        if case == "route":
            V = inputs.QWEN_V
            lut = torch.from_numpy(inputs.routing_lut(V, 0.3)).to(dev)
            for B in (64, 2048):
                ids = torch.from_numpy(inputs.token_ids_zipf(B, V, seed=inputs.SEED_IDS + B)).to(dev)
                perm = torch.empty(B, dtype=torch.int32, device=dev)
                nd = torch.empty(1, dtype=torch.int32, device=dev)
                st = torch.zeros(1, dtype=torch.int32, device=dev)
                for _ in range(n_calls):
                    sats.route(ids, lut, perm, nd, st, stream=stream)
                stream.synchronize()
                info["n_dense_%d" % B] = int(nd.item())
            ok = True
        elif case in ("batch64", "union", "lora", "small", "stack", "prefill"):
            H, N = (inputs.SMALL_H, inputs.SMALL_N) if case == "small" else (inputs.LLAMA_H, inputs.LLAMA_N)
            layer = sats.Layer(*inputs.mlp_weights_device(H, N), stream=stream)
            B = {"batch64": 64, "union": 8, "lora": 1, "small": 1, "stack": 64, "prefill": 2048}[case]
            k = {"batch64": 0.5, "union": 0.9, "lora": 0.7, "small": 0.5, "stack": 0.5, "prefill": 0.9}[case]
            t = threshold(layer, H, N, k)
            ws = sats.Workspace(H, N, B, device=dev, stream=stream)
            y = torch.empty(B, H, dtype=torch.float32, device=dev)
            idx = torch.empty(B, N, dtype=torch.int32, device=dev)
            cnt = torch.empty(B, dtype=torch.int32, device=dev)
            xb = torch.from_numpy(inputs.activations_bf16(B, H).view(np.int16)).to(dev)
            if case == "lora":
                r = 16
                ad = [torch.from_numpy(m.view(np.int16)).to(dev) for m in inputs.lora_adapter(H, N, r)]
                lora = sats.Lora(layer, *ad, scale=1.0, stream=stream)
                for _ in range(n_calls):
                    sats.sparse_mlp_lora(layer, lora, xb, t, y, ws, idx, cnt, stream=stream)
            elif case == "union":
                for _ in range(n_calls):
                    sats.sparse_mlp_union(layer, xb, t, y, ws, idx, cnt, stream=stream)
            elif case in ("stack", "prefill"):
                V = inputs.LLAMA_V
                lut = torch.from_numpy(inputs.routing_lut(V, 0.2, seed=inputs.SEED_LUT + 5)).to(dev)
                ids = torch.from_numpy(inputs.token_ids_zipf(B, V, seed=inputs.SEED_IDS + B)).to(dev)
                nw = torch.from_numpy(inputs.norm_weight(H)).to(dev)
                x = torch.from_numpy(inputs.activations_f32(B, H)).to(dev)
                for _ in range(n_calls):
                    sats.mlp_stack([layer], [nw], [t], 1e-5, x, ws, token_ids=ids, lut=lut, stream=stream)
            else:
                for _ in range(n_calls):
                    sats.sparse_mlp(layer, xb, t, y, ws, idx, cnt, stream=stream)
            stream.synchronize()
            ok = sats.get_error(ws, stream=stream) == sats.OK
            info.update({"hidden": H, "intermediate": N, "tokens": B, "target_sparsity": k,
                         "tensor_cores": sats.uses_tensor_cores(H, B)})
            if case not in ("stack", "prefill"):
                info["kept_token0"] = int(cnt[0].item())
            if case == "lora":
                lora.close()
            layer.close()
        else:
            raise SystemExit("unknown profile case " + case)
    info["status_ok"] = ok
    print(json.dumps(info))
    if not ok:
        raise RuntimeError("device status after the profile case")


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="sats", choices=["sats", "reference"])
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-batched", action="store_true", help="skip the batched tensor-core measurements")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the compact measurements of the other four workloads in the headline line")
    ap.add_argument("--workload", default=WORKLOAD, choices=sorted(inputs.WORKLOADS),
                    help="the headline workload (default) or one of the other four, reported on their own line")
    ap.add_argument("--profile-batch", type=int, default=0,
                    help="small capture case for ncu: `warmup + steps` calls at this batch size on one layer copy")
    ap.add_argument("--profile", action="store_true",
                    help="small capture case for ncu: one layer copy, timed calls only, no CPU baseline")
    ap.add_argument("--profile-case", default="", choices=("",) + PROFILE_CASES,
                    help="small capture case for ncu of one kernel group (see run_profile_case)")
    args = ap.parse_args()
    if args.profile_case:
        run_profile_case(args)
        return
    if args.profile or args.profile_batch:
        args.no_cpu_baseline = True
        args.no_batched = True
        args.no_configs = True
    if args.impl == "reference":
        run_reference(args)
    elif args.workload != WORKLOAD:
        run_workload(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
