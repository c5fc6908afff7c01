"""Throughput of the three-stage attention path (prefill, prefill_kv, decode) on GB300.

One step = one pass of the whole hot path over the long-context workload (batch 1,
40 query heads, 8 KV heads, head_dim 128, RoPE theta 1e6, static max length
32768): prefill of 4096 tokens, prefill_kv of a 4096-token chunk over 28672
history tokens, and one decode step at 32767 valid tokens, all on one KV cache.
Inputs are seeded synthetic bf16 N(0,1)/sqrt(128) values (synthetic/), resident in
HBM before the timed region; L2 is flushed between steps by a 256 MB write followed
by a 256 MB read of another buffer, so that no line of the step's inputs and no dirty
line (whose write-back the next kernel would pay for) is left in L2.

value     algorithmic attention FLOP of the step (4*D per unmasked query-key pair
          per query head, exact causal count) / mean device step time, TFLOP/s.
e2e       the same metric through the same C-ABI calls with host buffers: every
          step copies its q/k/v from pinned host memory and its outputs back
          (copies on their own streams, overlapping the neighbouring steps' compute).
roofline  the dominant kernel (flash_fwd) against the measured sustained bf16 tensor peak
          (it is timed inside the step loop; the burst-peak fraction is given beside it).
stages    per-stage times; prefill stages in TFLOP/s (fraction of the sustained peak),
          decode in HBM GB/s; each prefill stage's kernels also called alone (up to 20 calls,
          L2 flushed before each) with the flash kernel's rate against the burst peak.
configs   every configuration's stage on its own (7B-class prefill 512, prefill_kv 512 over
          1536, the decode sweep, the long-context stages): median of CUDA-event-timed calls
          with L2 flushed before each, TFLOP/s or GB/s and the fraction of the measured peak.
          (value comes from a pass with one event pair per step; stages, per-kernel
          times and the roofline from a second, instrumented pass over the same steps.)
cpu_baseline  the CPU oracle on a bounded row sample of the same step.

--impl reference times the CPU oracle (the reference arm of this path) instead.
--sweep times every configuration's stages, the stage driver, decode loops, the
multi-token decode, the W4BF16 decode GEMV and decode block; --stage / --w4 M,N,K /
--layer B,HIST only run one stage, GEMV shape or decode block (the launch pattern of a
profiler capture).
Multi-GPU (torchrun): every rank runs its own replica of the workload (weak
scaling, no collective on the data path); value is the whole-job aggregate.
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
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from synthetic import gen  # noqa: E402
from synthetic import workloads as w  # noqa: E402

METRIC = "prefill/prefill_kv attn TFLOP/s; decode KV GB/s; % of GB300 roofline"
WORKLOAD = ("long-context three-stage step: B1 Hq40 Hkv8 D128 theta1e6 L32768; prefill 4096 + "
            "prefill_kv 4096 over 28672 + decode at 32767")
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


# ----------------------------------------------------------------------------- work accounting


def prefill_pairs(hist: int, chunk: int) -> int:
    """Unmasked (query, key) pairs of one head: row i sees hist + i + 1 keys."""
    return chunk * hist + chunk * (chunk + 1) // 2


def attn_flops(shape, pairs_per_head: int) -> float:
    return 4.0 * shape.head_dim * shape.n_q_heads * shape.batch * pairs_per_head


def decode_bytes(shape, hist: int) -> float:
    """Algorithmic HBM bytes of one decode step per sequence: the K/V history read once,
    q and the new k/v read, the new k/v written to the cache, out written (bf16)."""
    d, hq, hkv = shape.head_dim, shape.n_q_heads, shape.n_kv_heads
    return shape.batch * (hist * hkv * d * 2 * 2 + hq * d * 2 * 2 + hkv * d * 2 * 4)


S = w.LONG
STAGES = {
    "prefill": dict(hist=0, chunk=w.LONG_PREFILL),
    "prefill_kv": dict(hist=w.LONG_PKV_HIST, chunk=w.LONG_PKV_CHUNK),
    "decode": dict(hist=w.LONG_DECODE_HIST, chunk=1),
}
FLOPS = {k: attn_flops(S, prefill_pairs(v["hist"], v["chunk"])) for k, v in STAGES.items()}
STEP_FLOPS = sum(FLOPS.values())
DECODE_BYTES = decode_bytes(S, w.LONG_DECODE_HIST)


# ----------------------------------------------------------------------------- helpers


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def dist_env():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("LOCAL_RANK", 0)), int(os.environ.get("WORLD_SIZE", 1))


def max_over_ranks(x: float, dist, device) -> float:
    """The maximum of x over all ranks (x itself without a process group)."""
    if dist is None:
        return x
    import torch
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_tflops(world: int, ms: float) -> float:
    """Whole-job throughput: each of `world` ranks ran one replica of the step (weak
    scaling, no exchange); the slowest rank's step time counts."""
    return world * STEP_FLOPS / (ms * 1e-3) / 1e12


def make_inputs():
    """Seeded host inputs of the step (bf16 bit patterns)."""
    data = {}
    for name, st in STAGES.items():
        data[name] = w.tokens(S, f"bench_{name}", st["chunk"])
    kc, vc = w.cache(S, "bench_history", w.LONG_PKV_HIST, fill="zero")
    return data, kc, vc


class ClockSampler:
    """nvidia-smi clock / throttle-reason samples while the timed region runs."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.dev = device_index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                                          "-lms", "100", "-i", str(self.dev)], stdout=subprocess.PIPE,
                                         stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, smax, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for line in out.strip().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def flash_traffic_from_profile():
    """DRAM bytes per flash_fwd-kind launch (dram__bytes_read + dram__bytes_write of one
    step's flash launches, from the committed single-pass ncu capture, divided by the
    launches per step), if that capture was taken on the current kernel source (its
    sha256 is recorded there); else None."""
    path = os.path.join(ROOT, "profiles", "flash_fwd_long_step.md")
    src = os.path.join(ROOT, "paper_2607_15865_gb300", "csrc", "flash_fwd.cu")
    if not os.path.exists(path):
        return None
    sha = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
    kv = {}
    for line in open(path):
        if line.startswith("- ") and ":" in line:
            k, v = line[2:].split(":", 1)
            kv[k.strip()] = v.strip().strip("`")
    if kv.get("kernel_source_sha256_16") != sha:
        return None
    try:
        return float(kv["dram_bytes_per_step_full_size"]) / int(kv["flash_launches_per_step"])
    except (KeyError, ValueError, ZeroDivisionError):
        return None


# ----------------------------------------------------------------------------- oracle sample


def oracle_sample(data, kc0, vc0, rows_pkv: int, rows_prefill: int, seed: int = 7, threads: int = 1):
    """Runs the oracle over a bounded row sample of one step (append every stage's new
    tokens in order, then the sampled rows of each stage, on `threads` host cores).
    Returns (rows, outputs, algorithmic FLOP of the sampled rows, seconds)."""
    from oracle import oracle as O
    rng = np.random.default_rng(seed)
    kc, vc = kc0.copy(), vc0.copy()
    picks = {"prefill": rows_prefill, "prefill_kv": rows_pkv, "decode": S.n_q_heads}
    rows, outs, flops = {}, {}, 0.0
    t0 = time.perf_counter()
    for name, st in STAGES.items():
        q, k, v = data[name]
        O.append(S, k, v, st["hist"], kc, vc)
        n = picks[name]
        if name == "decode":
            r = np.array([(0, 0, h) for h in range(S.n_q_heads)], np.int32)
        else:
            r = np.stack([np.zeros(n, np.int64), rng.integers(0, st["chunk"], n),
                          rng.integers(0, S.n_q_heads, n)], 1).astype(np.int32)
        outs[name] = O.attend_rows_parallel(S, q, st["hist"], kc, vc, r, threads=threads)
        rows[name] = r
        flops += float(sum(4.0 * S.head_dim * (st["hist"] + int(i) + 1) for i in r[:, 1]))
    return rows, outs, flops, time.perf_counter() - t0


# ----------------------------------------------------------------------------- reference arm


def run_reference(args):
    rank, _, world = dist_env()
    if rank != 0:
        return 0
    data, kc, vc = make_inputs()
    oracle_sample(data, kc, vc, 2, 2)  # build + warm the oracle library
    ncores = os.cpu_count() or 1
    n_pkv, n_pf = args.ref_rows * ncores, max(1, args.ref_rows // 4) * ncores
    times, flops = [], []
    for _ in range(args.warmup):
        oracle_sample(data, kc, vc, n_pkv, n_pf, threads=ncores)
    for i in range(args.steps):
        _, _, f, t = oracle_sample(data, kc, vc, n_pkv, n_pf, seed=100 + i, threads=ncores)
        times.append(t)
        flops.append(f)
    value = sum(flops) / sum(times) / 1e12
    sample = (f"per step {n_pkv} prefill_kv rows + {n_pf} prefill rows + {S.n_q_heads} decode rows of the "
              f"workload on {ncores} threads, all new tokens appended")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * sum(times) / len(times),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": WORKLOAD, "sample": sample},
            "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": ncores, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ----------------------------------------------------------------------------- our arm


def run_ours(args):
    import torch

    rank, local_rank, world = dist_env()
    dist = None
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        dist.init_process_group(backend=backend)
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)

    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_15865_gb300.attention import Attention

    data, kc_h, vc_h = make_inputs()
    d = {name: tuple(torch.from_numpy(a.view(np.int16)).to(dev) for a in arrs) for name, arrs in data.items()}
    kc = torch.from_numpy(kc_h.view(np.int16)).to(dev)
    vc = torch.from_numpy(vc_h.view(np.int16)).to(dev)
    hist_dec = torch.full((S.batch,), STAGES["decode"]["hist"], dtype=torch.int32, device=dev)
    outs = {name: torch.empty_like(d[name][0]) for name in STAGES}
    flush_w = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    flush_r = torch.ones(256 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)

    def l2_flush():
        flush_w.zero_()
        flush_r.sum()

    attn = Attention.for_shape(S)
    stream = torch.cuda.current_stream()

    def step(src=None, dst=None):
        qkv = d if src is None else src
        o = outs if dst is None else dst
        attn.prefill(*qkv["prefill"], kc, vc, out=o["prefill"], stream=stream)
        attn.prefill_kv(*qkv["prefill_kv"], STAGES["prefill_kv"]["hist"], kc, vc, out=o["prefill_kv"],
                        stream=stream)
        attn.decode(*qkv["decode"], hist_dec, kc, vc, out=o["decode"], stream=stream)

    for _ in range(args.warmup):
        l2_flush()
        step()
    torch.cuda.synchronize()
    if attn.device_error() != 0:
        raise RuntimeError("device error word set during warm-up")

    # ------------------------------------------------------------ timed region (device-resident inputs)
    # Loop A times the step with one event pair per step and nothing else inside it: the
    # headline value.  Loop B repeats the same K steps with an event pair around every
    # stage and the library's own pair around every kernel launch (its kernel timing),
    # for the per-stage times and the roofline of the dominant kernel.  (Those 16 event
    # records per step cost 1-2% of the step, which is why they stay out of loop A.)
    K = args.steps
    ev_a = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(K)]
    sampler = ClockSampler(local_rank)
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    sampler.start()
    time.sleep(0.3)  # let the sampler start before the GPU gets busy
    for i in range(K):
        l2_flush()
        ev_a[i][0].record(stream)
        step()
        ev_a[i][1].record(stream)
    torch.cuda.synchronize()
    if dist is not None:
        dist.barrier()
    step_ms = [a.elapsed_time(b) for a, b in ev_a]
    ms = max_over_ranks(sum(step_ms) / K, dist, dev)

    attn.timing_read()
    attn.timing_enable(8 * K)
    for i in range(K):
        l2_flush()
        ev[i][0].record(stream)
        attn.prefill(*d["prefill"], kc, vc, out=outs["prefill"], stream=stream)
        ev[i][1].record(stream)
        attn.prefill_kv(*d["prefill_kv"], STAGES["prefill_kv"]["hist"], kc, vc, out=outs["prefill_kv"], stream=stream)
        ev[i][2].record(stream)
        attn.decode(*d["decode"], hist_dec, kc, vc, out=outs["decode"], stream=stream)
        ev[i][3].record(stream)
    torch.cuda.synchronize()
    kern = attn.timing_read()
    attn.timing_enable(0)
    stage_ms = {name: sum(ev[i][j].elapsed_time(ev[i][j + 1]) for i in range(K)) / K
                for j, name in enumerate(STAGES)}
    # Each prefill stage's kernels on their own (library kernel timing, L2 flushed before every
    # call), so that the flash kernel's share of a stage is reported beside the stage.
    stage_kern = {}
    n_alone = min(K, 20)
    for name in ("prefill", "prefill_kv"):
        attn.timing_read()
        attn.timing_enable(4 * n_alone)
        for _ in range(n_alone):
            l2_flush()
            if name == "prefill":
                attn.prefill(*d["prefill"], kc, vc, out=outs["prefill"], stream=stream)
            else:
                attn.prefill_kv(*d["prefill_kv"], STAGES["prefill_kv"]["hist"], kc, vc, out=outs["prefill_kv"],
                                stream=stream)
        torch.cuda.synchronize()
        stage_kern[name] = {k: v[0] / n_alone for k, v in attn.timing_read().items() if v[1] > 0}
        attn.timing_enable(0)
    if attn.device_error() != 0:
        raise RuntimeError("device error word set during the timed region")

    # ------------------------------------------------------------ end to end (host buffers)
    # Every step copies its own q/k/v from pinned host memory and reads its own outputs
    # back, through the same C-ABI calls.  As a serving loop would, the copies run on
    # their own streams into double-buffered device tensors, so step i+1's inputs go up
    # and step i-1's outputs come down while step i computes; the steps stay ordered on
    # the compute stream through the cache.  No L2 flush here: each step's 117 MB of
    # inputs arrive by copy and its caches (134 MB) and inputs together exceed L2.
    host = {name: tuple(torch.from_numpy(a.view(np.int16)).pin_memory() for a in arrs) for name, arrs in data.items()}
    host_out = {name: torch.empty(tuple(outs[name].shape), dtype=torch.int16).pin_memory() for name in STAGES}
    h2d = sum(t.numel() * 2 for arrs in host.values() for t in arrs)
    d2h = sum(t.numel() * 2 for t in host_out.values())
    d_sets = [d, {name: tuple(torch.empty_like(t) for t in arrs) for name, arrs in d.items()}]
    o_sets = [outs, {name: torch.empty_like(t) for name, t in outs.items()}]
    copy_in, copy_out = torch.cuda.Stream(), torch.cuda.Stream()
    ev_in = [torch.cuda.Event() for _ in range(K)]
    ev_done = [torch.cuda.Event() for _ in range(K)]
    ev_out = [torch.cuda.Event() for _ in range(K)]
    e2e_start, e2e_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e2e_start.record(stream)
    copy_in.wait_event(e2e_start)
    for i in range(K):
        si = i % 2
        with torch.cuda.stream(copy_in):
            if i >= 2:
                copy_in.wait_event(ev_done[i - 2])  # the compute of step i-2 has read this set
            for name in STAGES:
                for dst, src in zip(d_sets[si][name], host[name]):
                    dst.copy_(src, non_blocking=True)
            ev_in[i].record(copy_in)
        stream.wait_event(ev_in[i])
        if i >= 2:
            stream.wait_event(ev_out[i - 2])  # step i-2's outputs in this set are read back
        step(src=d_sets[si], dst=o_sets[si])
        ev_done[i].record(stream)
        with torch.cuda.stream(copy_out):
            copy_out.wait_event(ev_done[i])
            for name in STAGES:
                host_out[name].copy_(o_sets[si][name], non_blocking=True)
            ev_out[i].record(copy_out)
    stream.wait_event(ev_out[K - 1])
    e2e_end.record(stream)
    torch.cuda.synchronize()
    clocks = sampler.stop()
    e2e_ms = max_over_ranks(e2e_start.elapsed_time(e2e_end) / K, dist, dev)

    # ------------------------------------------------------------ the other configurations, stage by stage
    # (after the timed step: CUDA events around each stage call, L2 flushed before each)
    cfg_rows = None
    if rank == 0 and not args.no_configs:
        cfg_rows, _, _, _ = config_rows(dev, args.config_reps, graphs=False)

    # ------------------------------------------------------------ parity of the timed outputs + CPU baseline
    result = {}
    if rank == 0:
        peaks, peak_kind = load_peaks()
        got = {name: outs[name].cpu().numpy().view(np.uint16) for name in STAGES}
        cpu = None
        parity = {}
        rows, ref, f_cpu, t_cpu = oracle_sample(data, kc_h, vc_h, args.cpu_rows, max(1, args.cpu_rows // 4))
        for name in STAGES:
            r = rows[name]
            g = gen.bf16_bits_to_f32(got[name][r[:, 0], r[:, 1], r[:, 2]]).astype(np.float64)
            e = gen.bf16_bits_to_f32(ref[name]).astype(np.float64)
            err = np.abs(g - e)
            rel = float(np.linalg.norm(g - e) / max(np.linalg.norm(e), 1e-30))
            parity[name] = {"rows": int(len(r)), "max_abs": float(err.max()), "mean_abs": float(err.mean()),
                            "rel": rel}
            if not (err.max() <= 2e-2 and err.mean() <= 2e-3 and rel <= 1e-2 and np.isfinite(g).all()):
                raise SystemExit(f"parity check failed for {name}: {parity[name]}")
        if world == 1 and not args.no_cpu_baseline:
            # the same oracle on every host core (whole rows per thread), on a sample
            # that many times larger, beside the single-core figure above
            ncores = os.cpu_count() or 1
            _, _, f_all, t_all = oracle_sample(data, kc_h, vc_h, args.cpu_rows * ncores,
                                               max(1, args.cpu_rows // 4) * ncores, seed=11, threads=ncores)
            cpu = {"value": f_all / t_all / 1e12, "unit": "TFLOP/s", "cores": ncores, "kind": "oracle",
                   "sample": (f"{args.cpu_rows * ncores} prefill_kv rows + {max(1, args.cpu_rows // 4) * ncores} "
                              f"prefill rows + {S.n_q_heads} decode rows of the step, {ncores} threads, "
                              f"{t_all:.1f} s"),
                   "one_core": {"value": f_cpu / t_cpu / 1e12, "unit": "TFLOP/s", "cores": 1,
                                "sample": (f"{args.cpu_rows} prefill_kv rows + {max(1, args.cpu_rows // 4)} "
                                           f"prefill rows + {S.n_q_heads} decode rows, single-threaded, "
                                           f"{t_cpu:.1f} s")}}
        value = job_tflops(world, ms)
        flash_ms = kern["flash_fwd"][0]
        flash_n = kern["flash_fwd"][1]
        flash_flops = (FLOPS["prefill"] + FLOPS["prefill_kv"]) * K
        flash_tflops = flash_flops / (flash_ms * 1e-3) / 1e12
        tc_peak = float(peaks["bf16_tflops"])
        # flash_fwd is timed inside the K-step loop (seconds of back-to-back tensor work under
        # the power cap): its roofline is the sustained dense bf16 figure; the burst one (a
        # kernel timed alone, as the per-configuration rows are) is reported beside it.
        tc_sustained = float(peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"]))
        traffic = flash_traffic_from_profile()
        hbm = float(peaks["hbm_gbs"])
        stages = {}
        for name in STAGES:
            t_s = stage_ms[name] * 1e-3
            if name == "decode":
                gbs = DECODE_BYTES / t_s / 1e9
                stages[name] = {"ms": stage_ms[name], "GB/s": gbs, "frac_hbm": gbs / hbm,
                                "kernel_ms": {k: kern[k][0] / K for k in ("decode_split", "decode_combine")}}
            else:
                tf = FLOPS[name] / t_s / 1e12
                # the flash kernel alone (called by itself): against the burst peak, as a
                # kernel timed alone is
                tk = FLOPS[name] / (stage_kern[name]["flash_fwd"] * 1e-3) / 1e12
                stages[name] = {"ms": stage_ms[name], "TFLOP/s": tf, "frac_tensor": tf / tc_sustained,
                                "kernel_ms_alone": stage_kern[name], "flash_TFLOP/s_alone": tk,
                                "flash_frac_of_burst_alone": tk / tc_peak}
        launches = int(sum(n for _, n in kern.values()))
        result = {
            "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world, "steps": K,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": WORKLOAD, "l2": "flushed between steps (256 MB write + 256 MB read, untimed)",
                       "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
                       "step_gflop": STEP_FLOPS / 1e9},
            "roofline": {"bound": "tensor", "achieved": flash_tflops, "peak": tc_sustained, "unit": "TFLOP/s",
                         "frac": flash_tflops / tc_sustained, "traffic": traffic, "kernel": "flash_fwd",
                         "peak_source": f"{peak_kind} bf16_tflops_sustained (timed inside the {K}-step loop)",
                         "frac_of_burst_peak": flash_tflops / tc_peak, "burst_peak": tc_peak,
                         "launch_ms_avg": flash_ms / max(flash_n, 1)},
            "stages": stages,
            "kernels_ms_per_step": {k: v[0] / K for k, v in kern.items()},
            "cpu_baseline": cpu,
            "e2e": {"value": job_tflops(world, e2e_ms), "unit": "TFLOP/s",
                    "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms,
                    "copies": "pinned host, own streams, overlapping the neighbouring steps",
                    "l2": "not flushed: each step's inputs arrive by copy; inputs + caches exceed L2"},
            "configs": cfg_rows,
            "gpu_launches": launches,
            "clocks": clocks,
            "parity": parity,
        }
        print(json.dumps(result), flush=True)
    attn.close()
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()
    return 0


# ----------------------------------------------------------------------------- per-config sweep


def config_rows(dev, reps: int, graphs: bool):
    """Per-configuration stage rows (the paper's workloads: 7B-class prefill 512, prefill_kv
    512 over 1536, the decode sweep B in {1,4,16} x hist in {1024, 4096, 8191}, and the
    long-context stages one by one).  Each row is the median of `reps` calls timed with CUDA
    events around the stage call, inputs resident, L2 flushed (256 MB write + 256 MB read)
    before every call and a short GPU sleep in front of it, so the host's launch cost stays
    outside the events.  CUDA events on a GB300 tick in steps of 2.048 us and read about
    4.5 us around an empty kernel, which dominates the small rows; so every row also has
    `loop_ms`: the same call replayed 10 times from one CUDA graph, each time after the L2
    flush, less the same graph with the flushes alone, per call (the rates in `loop_*`).
    graphs: also time each decode step replayed from a CUDA graph."""
    import torch
    from paper_2607_15865_gb300.attention import Attention
    from synthetic.workloads import Shape
    flush_w = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    flush_r = torch.ones(256 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    peaks, _ = load_peaks()
    tc_peak, hbm = float(peaks["bf16_tflops"]), float(peaks["hbm_gbs"])

    def rnd(shape, gen):
        return (torch.randn(*shape, device=dev, generator=gen) * 0.0884).to(torch.bfloat16)

    def time_calls(fn, reps):
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(reps)]
        for _ in range(3):
            flush_w.zero_()
            flush_r.sum()
            fn()
        for a, b in evs:
            flush_w.zero_()
            flush_r.sum()
            torch.cuda._sleep(200_000)  # keeps the GPU busy while the host issues fn()
            a.record()
            fn()
            b.record()
        torch.cuda.synchronize()
        return sorted(a.elapsed_time(b) for a, b in evs)[reps // 2]  # median, ms

    def loop_ms(fn, n=10):
        # per call, in a CUDA graph of n (L2 flush, call) pairs, less the flushes alone (ms)
        t = []
        for with_call in (False, True):
            side = torch.cuda.Stream()
            side.wait_stream(torch.cuda.current_stream())
            gr = torch.cuda.CUDAGraph()
            with torch.cuda.stream(side), torch.cuda.graph(gr, stream=side):
                for _ in range(n):
                    flush_w.zero_()
                    flush_r.sum()
                    if with_call:
                        fn()
            torch.cuda.current_stream().wait_stream(side)
            gr.replay()
            torch.cuda.synchronize()
            ts = []
            for _ in range(5):
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record()
                gr.replay()
                b.record()
                torch.cuda.synchronize()
                ts.append(a.elapsed_time(b))
            t.append(sorted(ts)[2])
            del gr
        return max(t[1] - t[0], 0.0) / n

    rows = []
    gen = torch.Generator(device=dev).manual_seed(1)
    cases = [("7B prefill 512", w.PREFILL_7B, 0, 512),
             ("prefill_kv 512 over 1536", w.PREFILL_KV, 1536, 512),
             ("long prefill 4096", S, 0, w.LONG_PREFILL),
             ("long prefill_kv 4096 over 28672", S, w.LONG_PKV_HIST, w.LONG_PKV_CHUNK)]
    for name, sh, hist, chunk in cases:
        attn = Attention.for_shape(sh)
        q = rnd((sh.batch, chunk, sh.n_q_heads, sh.head_dim), gen)
        k = rnd((sh.batch, chunk, sh.n_kv_heads, sh.head_dim), gen)
        v = rnd((sh.batch, chunk, sh.n_kv_heads, sh.head_dim), gen)
        kc = rnd((sh.batch, sh.n_kv_heads, sh.max_len, sh.head_dim), gen)
        vc = rnd((sh.batch, sh.n_kv_heads, sh.max_len, sh.head_dim), gen)
        out = torch.empty_like(q)
        ms = time_calls(lambda: attn.prefill_kv(q, k, v, hist, kc, vc, out), reps)
        lms = loop_ms(lambda: attn.prefill_kv(q, k, v, hist, kc, vc, out))
        fl = attn_flops(sh, prefill_pairs(hist, chunk))
        tf, ltf = fl / (ms * 1e-3) / 1e12, fl / (lms * 1e-3) / 1e12
        rows.append({"config": name, "ms": ms, "TFLOP/s": tf, "frac_tensor": tf / tc_peak,
                     "loop_ms": lms, "loop_TFLOP/s": ltf, "loop_frac_tensor": ltf / tc_peak})
        attn.close()
    for bsz in w.DECODE_BATCHES:
        sh = w.decode_shape(bsz)
        attn = Attention.for_shape(sh)
        nbuf = max(2, int(2 * 130e6 // (sh.batch * sh.n_kv_heads * sh.max_len * sh.head_dim * 4)) + 1)
        caches = [(rnd((sh.batch, sh.n_kv_heads, sh.max_len, sh.head_dim), gen),
                   rnd((sh.batch, sh.n_kv_heads, sh.max_len, sh.head_dim), gen)) for _ in range(min(nbuf, 8))]
        q = rnd((sh.batch, 1, sh.n_q_heads, sh.head_dim), gen)
        k = rnd((sh.batch, 1, sh.n_kv_heads, sh.head_dim), gen)
        v = rnd((sh.batch, 1, sh.n_kv_heads, sh.head_dim), gen)
        out = torch.empty_like(q)
        for hist in w.DECODE_HISTS:
            hl = torch.full((sh.batch,), hist, dtype=torch.int32, device=dev)
            it = [0]

            def call():
                kc, vc = caches[it[0] % len(caches)]
                it[0] += 1
                attn.decode(q, k, v, hl, kc, vc, out)
            ms = time_calls(call, reps)
            lms = loop_ms(call)
            gbs, lgbs = decode_bytes(sh, hist) / (ms * 1e-3) / 1e9, decode_bytes(sh, hist) / (lms * 1e-3) / 1e9
            row = {"config": f"decode B{bsz} hist {hist}", "ms": ms, "GB/s": gbs, "frac_hbm": gbs / hbm,
                   "loop_ms": lms, "loop_GB/s": lgbs, "loop_frac_hbm": lgbs / hbm}
            rows.append(row)
            if not graphs:
                continue
            # the same step replayed from a CUDA graph (one graph per cache pair): what a
            # serving loop that captures its decode step sees
            grs = []
            for kc, vc in caches:
                attn.decode(q, k, v, hl, kc, vc, out)  # tensor maps built outside the capture
                gr = torch.cuda.CUDAGraph()
                side = torch.cuda.Stream()
                side.wait_stream(torch.cuda.current_stream())
                with torch.cuda.stream(side), torch.cuda.graph(gr, stream=side):
                    attn.decode(q, k, v, hl, kc, vc, out)
                torch.cuda.current_stream().wait_stream(side)
                grs.append(gr)
            torch.cuda.synchronize()
            git = [0]

            def replay():
                grs[git[0] % len(grs)].replay()
                git[0] += 1
            ms_g = time_calls(replay, reps)
            row["graph_ms"], row["graph_GB/s"] = ms_g, decode_bytes(sh, hist) / (ms_g * 1e-3) / 1e9
            del grs
        attn.close()
    # a batch of 16 with lengths spread over 64 .. 8191 (seeded): the split counts follow the
    # lengths, so the byte rate should stay near the uniform batch's
    sh = w.decode_shape(16)
    attn = Attention.for_shape(sh)
    kc = rnd((sh.batch, sh.n_kv_heads, sh.max_len, sh.head_dim), gen)
    vc = rnd((sh.batch, sh.n_kv_heads, sh.max_len, sh.head_dim), gen)
    q = rnd((sh.batch, 1, sh.n_q_heads, sh.head_dim), gen)
    k = rnd((sh.batch, 1, sh.n_kv_heads, sh.head_dim), gen)
    v = rnd((sh.batch, 1, sh.n_kv_heads, sh.head_dim), gen)
    out = torch.empty_like(q)
    lens = np.random.default_rng(16).integers(64, 8192, sh.batch).astype(np.int32)
    hl = torch.from_numpy(lens).to(dev)
    ms = time_calls(lambda: attn.decode(q, k, v, hl, kc, vc, out), reps)
    lms = loop_ms(lambda: attn.decode(q, k, v, hl, kc, vc, out))
    one = Shape("one", 1, sh.n_q_heads, sh.n_kv_heads, sh.head_dim, sh.max_len, sh.rope_theta)
    byts = sum(decode_bytes(one, int(h)) for h in lens)
    gbs, lgbs = byts / (ms * 1e-3) / 1e9, byts / (lms * 1e-3) / 1e9
    rows.append({"config": f"decode B16 lengths spread over 64..8191 (mean {int(lens.mean())})", "ms": ms,
                 "GB/s": gbs, "frac_hbm": gbs / hbm, "loop_ms": lms, "loop_GB/s": lgbs,
                 "loop_frac_hbm": lgbs / hbm})
    attn.close()
    del kc, vc
    attn = Attention.for_shape(S)
    kc = rnd((1, 8, 32768, 128), gen)
    vc = rnd((1, 8, 32768, 128), gen)
    q, k, v = rnd((1, 1, 40, 128), gen), rnd((1, 1, 8, 128), gen), rnd((1, 1, 8, 128), gen)
    out = torch.empty_like(q)
    hl = torch.full((1,), w.LONG_DECODE_HIST, dtype=torch.int32, device=dev)
    ms = time_calls(lambda: attn.decode(q, k, v, hl, kc, vc, out), reps)
    lms = loop_ms(lambda: attn.decode(q, k, v, hl, kc, vc, out))
    gbs, lgbs = DECODE_BYTES / (ms * 1e-3) / 1e9, DECODE_BYTES / (lms * 1e-3) / 1e9
    rows.append({"config": "long decode hist 32767", "ms": ms, "GB/s": gbs, "frac_hbm": gbs / hbm,
                 "loop_ms": lms, "loop_GB/s": lgbs, "loop_frac_hbm": lgbs / hbm})
    attn.close()
    del kc, vc
    return rows, time_calls, rnd, gen


def run_sweep(args):
    """Times every configuration's stage on one GPU (CUDA events around the stage call,
    inputs resident, L2 flushed before each timed call) and writes a table to
    --sweep-out; the default JSON line is not printed in this mode."""
    import torch

    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_15865_gb300.attention import Attention
    from synthetic.workloads import Shape
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    peaks, kind = load_peaks()
    tc_peak, hbm = float(peaks["bf16_tflops"]), float(peaks["hbm_gbs"])
    rows, time_calls, rnd, gen = config_rows(dev, args.sweep_reps, graphs=True)
    # The stage driver (Sections 4.1 and 4.5).  A 32768-token prompt as 1 prefill + 7
    # prefill_kv of 4096 tokens (the paper's 80K-prompt example scaled to this cache),
    # beside the same prompt in one prefill call.
    attn = Attention.for_shape(S)
    P, seg = S.max_len, w.LONG_PREFILL
    q = rnd((1, P, S.n_q_heads, S.head_dim), gen)
    k, v = rnd((1, P, S.n_kv_heads, S.head_dim), gen), rnd((1, P, S.n_kv_heads, S.head_dim), gen)
    kc, vc = torch.empty_like(k).view(1, S.n_kv_heads, P, S.head_dim), torch.empty_like(v).view(1, S.n_kv_heads, P, S.head_dim)
    out = torch.empty_like(q)
    flop = attn_flops(S, prefill_pairs(0, P))
    for name, sg in ((f"long prompt {P} as {P // seg} segments of {seg}", seg), (f"long prompt {P} in one prefill", P)):
        ms = time_calls(lambda: attn.prompt(q, k, v, 0, sg, kc, vc, out), max(3, args.sweep_reps // 4))
        tf = flop / (ms * 1e-3) / 1e12
        rows.append({"config": name, "ms": ms, "TFLOP/s": tf, "frac_tensor": tf / tc_peak})
    attn.close()
    del q, k, v, kc, vc, out
    # Decode loops of 32 steps per call from 4096 valid tokens (B16: bandwidth; B1: the
    # latency-bound case), each replayed from one CUDA graph: bytes = the 32 steps'
    # decode bytes.  Consecutive steps start as dependent launches.
    for bsz in (16, 1):
        sh = w.decode_shape(bsz)
        attn = Attention.for_shape(sh)
        n, hist = 32, 4096
        kc = rnd((sh.batch, sh.n_kv_heads, sh.max_len, sh.head_dim), gen)
        vc = rnd((sh.batch, sh.n_kv_heads, sh.max_len, sh.head_dim), gen)
        q = rnd((n, sh.batch, 1, sh.n_q_heads, sh.head_dim), gen)
        k = rnd((n, sh.batch, 1, sh.n_kv_heads, sh.head_dim), gen)
        v = rnd((n, sh.batch, 1, sh.n_kv_heads, sh.head_dim), gen)
        out = torch.empty_like(q)
        hl = torch.full((sh.batch,), hist, dtype=torch.int32, device=dev)
        attn.decode_steps(q, k, v, hl, kc, vc, out)
        gr = torch.cuda.CUDAGraph()
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side), torch.cuda.graph(gr, stream=side):
            attn.decode_steps(q, k, v, hl, kc, vc, out)
        torch.cuda.current_stream().wait_stream(side)
        torch.cuda.synchronize()
        ms = time_calls(gr.replay, args.sweep_reps)
        gbs = sum(decode_bytes(sh, hist + t) for t in range(n)) / (ms * 1e-3) / 1e9
        rows.append({"config": f"decode loop {n} steps B{bsz} from hist {hist} (CUDA graph)", "ms": ms,
                     "GB/s": gbs, "frac_hbm": gbs / hbm})
        attn.close()
        del kc, vc, q, k, v, out, gr
    # Multi-token decode (a speculative draft of n tokens verified in one call) against the
    # same n tokens as one prefill_kv chunk: bytes = the history's K/V read once plus the
    # new tokens' q, k, v and out.
    for sh, hist, n in ((w.decode_shape(1), 8188, 4), (S, w.LONG_DECODE_HIST - 2, 3), (w.decode_shape(1), 8184, 8),
                        (S, w.LONG_DECODE_HIST - 7, 8)):
        attn = Attention.for_shape(sh)
        kc = rnd((sh.batch, sh.n_kv_heads, sh.max_len, sh.head_dim), gen)
        vc = rnd((sh.batch, sh.n_kv_heads, sh.max_len, sh.head_dim), gen)
        q = rnd((sh.batch, n, sh.n_q_heads, sh.head_dim), gen)
        k = rnd((sh.batch, n, sh.n_kv_heads, sh.head_dim), gen)
        v = rnd((sh.batch, n, sh.n_kv_heads, sh.head_dim), gen)
        out = torch.empty_like(q)
        hl = torch.full((sh.batch,), hist, dtype=torch.int32, device=dev)
        byts = sh.batch * (hist * sh.n_kv_heads * sh.head_dim * 4 +
                           n * (sh.n_q_heads * sh.head_dim * 4 + sh.n_kv_heads * sh.head_dim * 8))
        tag = f"Hq{sh.n_q_heads} Hkv{sh.n_kv_heads} B{sh.batch} hist {hist}"
        for label, fn in ((f"verify {n} tokens, {tag}: multi-token decode",
                           lambda: attn.decode_multi(q, k, v, hl, kc, vc, out)),
                          (f"verify {n} tokens, {tag}: as a prefill_kv chunk",
                           lambda: attn.prefill_kv(q, k, v, hist, kc, vc, out))):
            ms = time_calls(fn, args.sweep_reps)
            gbs = byts / (ms * 1e-3) / 1e9
            rows.append({"config": label, "ms": ms, "GB/s": gbs, "frac_hbm": gbs / hbm})
        attn.close()
        del kc, vc
    # W4BF16 decode GEMV (the weight stream of the paper's W4BF16 decode): one large matrix
    # (268 MB of tiles, beyond L2) at 1 and 8 rows of x, and the 128 GEMVs of a 7B-class
    # decode step (32 layers x qkv, o, gate_up, down; 3.4 GB of tiles) replayed from one
    # CUDA graph.  Bytes = tiles + x + y.
    from paper_2607_15865_gb300.w4 import TILE_BYTES, w4bf16_gemv

    def w4_inputs(M, N, K):
        nrec = (N + 15) // 16 * (K // 128)
        tiles = torch.randint(0, 256, (nrec, TILE_BYTES), dtype=torch.uint8, device=dev, generator=gen)
        tiles[:, 1024:1056].view(torch.int16).fill_(0x3C00)  # scales 2^-7
        tiles[:, 1056:] &= 15
        x = rnd((M, K), gen)
        return tiles.view(-1), x, torch.empty((M, N), dtype=torch.bfloat16, device=dev)

    def w4_bytes(M, N, K):
        return (N + 15) // 16 * (K // 128) * TILE_BYTES + 2 * M * K + 2 * M * N

    for M in (1, 8):
        N, K = 65536, 8192
        tiles, x, y = w4_inputs(M, N, K)
        ms = time_calls(lambda: w4bf16_gemv(tiles, x, N, out=y, weights_static=True), args.sweep_reps)
        gbs = w4_bytes(M, N, K) / (ms * 1e-3) / 1e9
        rows.append({"config": f"W4BF16 GEMV M={M} N={N} K={K}", "ms": ms, "GB/s": gbs, "frac_hbm": gbs / hbm})
        del tiles, x, y
    layer = [(12288, 4096), (4096, 4096), (22016, 4096), (4096, 11008)]
    for M, early in ((1, False), (1, True), (4, True)):
        mats = [w4_inputs(M, N, K) + (N,) for N, K in layer * 32]
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            for tiles, x, y, N in mats:
                w4bf16_gemv(tiles, x, N, out=y, stream=side, weights_static=early)
        torch.cuda.synchronize()
        gr = torch.cuda.CUDAGraph()
        with torch.cuda.stream(side), torch.cuda.graph(gr, stream=side):
            for tiles, x, y, N in mats:
                w4bf16_gemv(tiles, x, N, out=y, stream=side, weights_static=early)
        torch.cuda.synchronize()
        ms = time_calls(gr.replay, args.sweep_reps)
        gbs = sum(w4_bytes(M, N, K) for N, K in layer * 32) / (ms * 1e-3) / 1e9
        tag = "weights streamed early" if early else "each GEMV after the previous"
        rows.append({"config": f"W4BF16 7B-class decode step M={M}: 128 GEMVs (CUDA graph, {tag})", "ms": ms,
                     "GB/s": gbs, "frac_hbm": gbs / hbm})
        del mats, gr
    # The prefill-side W4BF16 GEMM (attn_w4bf16_gemm) over a 4096-token chunk: the stacked QKV and
    # the o_proj of an 8B-class model; FLOP = 2 T N K.
    from paper_2607_15865_gb300.w4 import w4bf16_gemm
    for N, K in ((6144, 4096), (4096, 4096)):
        T = 4096
        tiles = w4_inputs(1, N, K)[0]
        x = rnd((T, K), gen)
        y = torch.empty((T, N), dtype=torch.bfloat16, device=dev)
        ms = time_calls(lambda: w4bf16_gemm(tiles, x, N, out=y), args.sweep_reps)
        tf = 2.0 * T * N * K / (ms * 1e-3) / 1e12
        rows.append({"config": f"W4BF16 GEMM T={T} N={N} K={K} (prefill projection)", "ms": ms, "TFLOP/s": tf,
                     "frac_tensor": tf / tc_peak})
        del tiles, x, y
    # The attention half of a decoder block with W4BF16 weights (attn_decode_layer: RMSNorm ->
    # stacked QKV GEMV -> decode attention -> o_proj + residual), 32 layers of an 8B-class
    # model (hidden 4096, Hq 32, Hkv 8, D 128) at 4096 valid tokens, one CUDA graph.  Bytes =
    # the weights' tile streams + the K/V history read + the new K/V and the activations.
    lsh = w.decode_shape(1)
    for bsz in (1, 4):
        sh = Shape(f"layer_b{bsz}", bsz, lsh.n_q_heads, lsh.n_kv_heads, lsh.head_dim, lsh.max_len, lsh.rope_theta)
        hidden, hist, nl = 4096, 4096, 32
        qd, kd = sh.n_q_heads * sh.head_dim, sh.n_kv_heads * sh.head_dim
        attn = Attention.for_shape(sh)
        gamma = (1.0 + 0.1 * torch.randn(hidden, device=dev, generator=gen)).to(torch.bfloat16)
        x = torch.randn(bsz, hidden, device=dev, generator=gen).to(torch.bfloat16)
        hl = torch.full((bsz,), hist, dtype=torch.int32, device=dev)
        layers_ = []
        for _ in range(nl):
            tq = w4_inputs(1, qd + 2 * kd, hidden)[0]
            to = w4_inputs(1, hidden, qd)[0]
            kc = rnd((sh.batch, sh.n_kv_heads, sh.max_len, sh.head_dim), gen)
            vc = rnd((sh.batch, sh.n_kv_heads, sh.max_len, sh.head_dim), gen)
            layers_.append((tq, to, kc, vc))

        def block_step(stream=None):
            h = x
            for tq, to, kc, vc in layers_:
                h = attn.decode_layer(h, gamma, 1e-6, tq, to, hl, kc, vc, weights_static=True, stream=stream)
            return h

        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            block_step(side)
        torch.cuda.synchronize()
        gr = torch.cuda.CUDAGraph()
        with torch.cuda.stream(side), torch.cuda.graph(gr, stream=side):
            block_step(side)
        torch.cuda.synchronize()
        ms = time_calls(gr.replay, args.sweep_reps)
        byts = nl * (w4_bytes(bsz, qd + 2 * kd, hidden) + w4_bytes(bsz, hidden, qd) +
                     decode_bytes(sh, hist) + 2 * bsz * hidden * 2)
        gbs = byts / (ms * 1e-3) / 1e9
        rows.append({"config": f"W4BF16 attention half of 32 decoder blocks B{bsz} hist {hist} (CUDA graph)",
                     "ms": ms, "GB/s": gbs, "frac_hbm": gbs / hbm})
        attn.close()
        del layers_, gr
    # The attention half of a decoder block over a prefill chunk (attn_prefill_layer: RMSNorm
    # pre-pass -> stacked QKV GEMM split into q, k, v -> RoPE + cache append + causal attention
    # -> o_proj GEMM + residual), the same 8B-class layer: a 4096-token prefill and a 4096-token
    # prefill_kv chunk over 4096 history tokens.  FLOP = the two projections (2 T N K each) + the
    # attention's 4 D per unmasked (query, key) pair per query head.
    lsh = w.decode_shape(1)
    hidden = 4096
    sh = Shape("prefill_layer", 1, lsh.n_q_heads, lsh.n_kv_heads, lsh.head_dim, lsh.max_len, lsh.rope_theta)
    qd, kd = sh.n_q_heads * sh.head_dim, sh.n_kv_heads * sh.head_dim
    attn = Attention.for_shape(sh)
    tq = w4_inputs(1, qd + 2 * kd, hidden)[0]
    to = w4_inputs(1, hidden, qd)[0]
    gamma = (1.0 + 0.1 * torch.randn(hidden, device=dev, generator=gen)).to(torch.bfloat16)
    kc = rnd((sh.batch, sh.n_kv_heads, sh.max_len, sh.head_dim), gen)
    vc = rnd((sh.batch, sh.n_kv_heads, sh.max_len, sh.head_dim), gen)
    for hist, n_tok in ((0, 4096), (4096, 4096)):
        x = torch.randn(1, n_tok, hidden, device=dev, generator=gen).to(torch.bfloat16)
        ws = torch.empty(attn.prefill_layer_workspace(hidden, n_tok), dtype=torch.uint8, device=dev)
        out = torch.empty_like(x)
        ms = time_calls(lambda: attn.prefill_layer(x, gamma, 1e-6, tq, to, hist, kc, vc, out=out, workspace=ws),
                        max(3, args.sweep_reps // 2))
        flop = 2.0 * n_tok * (qd + 2 * kd) * hidden + 2.0 * n_tok * hidden * qd + attn_flops(sh, prefill_pairs(hist, n_tok))
        tf = flop / (ms * 1e-3) / 1e12
        rows.append({"config": f"W4BF16 attention half of a decoder block, prefill chunk {n_tok} over {hist} "
                               f"(hidden {hidden}, Hq {sh.n_q_heads}, Hkv {sh.n_kv_heads})",
                     "ms": ms, "TFLOP/s": tf, "frac_tensor": tf / tc_peak})
        del x, ws, out
    attn.close()
    del tq, to, kc, vc
    doc = {"peaks": {"bf16_tflops": tc_peak, "hbm_gbs": hbm, "source": kind}, "rows": rows}
    with open(args.sweep_out, "w") as f:
        json.dump(doc, f, indent=1)
    for r in rows:
        extra = f"{r['TFLOP/s']:8.1f} TFLOP/s {100*r['frac_tensor']:5.1f}%" if "TFLOP/s" in r else \
            f"{r['GB/s']:8.1f} GB/s    {100*r['frac_hbm']:5.1f}%"
        if "loop_ms" in r:
            extra += f"   (flushed graph loop: {r['loop_ms']*1e3:6.1f} us)"
        if "graph_ms" in r:
            extra += f"   (CUDA graph: {r['graph_ms']*1e3:6.1f} us {r['graph_GB/s']:7.1f} GB/s)"
        print(f"{r['config']:36s} {r['ms']*1e3:9.1f} us {extra}", file=sys.stderr)
    return 0


# ----------------------------------------------------------------------------- one stage (profiling)


def run_stage(args):
    """Runs one stage of the long-context workload --warmup + --reps times on random
    device inputs (no timing, no JSON line): the launch pattern that profiler captures
    of a single kernel use.  --hist / --chunk override the stage's sizes; --shape 7b or
    pkv512 takes the 7B-class prefill (Hq28 Hkv4, 512 tokens) or the prefill_kv of 512
    tokens over 1536 (Hq32 Hkv8) instead."""
    import torch

    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_15865_gb300.attention import Attention
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    st = STAGES[args.stage]
    hist = st["hist"] if args.hist is None else args.hist
    chunk = st["chunk"] if args.chunk is None else args.chunk
    shape = S
    if args.shape == "7b":
        shape, hist, chunk = w.PREFILL_7B, 0, 512
    elif args.shape == "pkv512":
        shape, hist, chunk = w.PREFILL_KV, 1536, 512
    g = torch.Generator(device=dev).manual_seed(3)

    def rnd(*shape):
        return (torch.randn(*shape, device=dev, generator=g) * 0.0884).to(torch.bfloat16)

    attn = Attention.for_shape(shape)
    kc = rnd(shape.batch, shape.n_kv_heads, shape.max_len, shape.head_dim)
    vc = rnd(shape.batch, shape.n_kv_heads, shape.max_len, shape.head_dim)
    q = rnd(shape.batch, chunk, shape.n_q_heads, shape.head_dim)
    k = rnd(shape.batch, chunk, shape.n_kv_heads, shape.head_dim)
    v = rnd(shape.batch, chunk, shape.n_kv_heads, shape.head_dim)
    out = torch.empty_like(q)
    hl = torch.full((shape.batch,), hist, dtype=torch.int32, device=dev)
    for _ in range(args.warmup + args.reps):
        if args.stage == "decode":
            attn.decode(q, k, v, hl, kc, vc, out)
        else:
            attn.prefill_kv(q, k, v, hist, kc, vc, out)
    torch.cuda.synchronize()
    flags = attn.device_error()
    attn.close()
    print(f"stage {args.stage} hist {hist} chunk {chunk}: {args.warmup} + {args.reps} calls, device error word {flags}")
    return 0 if flags == 0 else 1


def run_w4_stage(args):
    """Runs the W4BF16 GEMV of --w4 M,N,K --warmup + --reps times on random tiles (no
    timing, no JSON line): the launch pattern of a profiler capture of that kernel."""
    import torch

    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_15865_gb300.w4 import TILE_BYTES, w4bf16_gemv
    M, N, K = (int(v) for v in args.w4.split(","))
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    g = torch.Generator(device=dev).manual_seed(3)
    tiles = torch.randint(0, 256, ((N + 15) // 16 * (K // 128), TILE_BYTES), dtype=torch.uint8, device=dev,
                          generator=g)
    tiles[:, 1024:1056].view(torch.int16).fill_(0x3C00)
    tiles[:, 1056:] &= 15
    x = (torch.randn(M, K, device=dev, generator=g)).to(torch.bfloat16)
    y = torch.empty((M, N), dtype=torch.bfloat16, device=dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    for _ in range(args.warmup + args.reps):
        w4bf16_gemv(tiles.view(-1), x, N, out=y, err=err)
    torch.cuda.synchronize()
    flags = int(err.item())
    print(f"w4 GEMV M={M} N={N} K={K}: {args.warmup} + {args.reps} calls, device error word {flags}")
    return 0 if flags == 0 else 1


def run_gemm_stage(args):
    """Runs the W4BF16 GEMM of --gemm T,N,K (T tokens, N features, K inputs) --warmup + --reps
    times on random tiles (no timing, no JSON line): the launch pattern of a profiler capture."""
    import torch

    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_15865_gb300.w4 import TILE_BYTES, w4bf16_gemm
    T, N, K = (int(v) for v in args.gemm.split(","))
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    g = torch.Generator(device=dev).manual_seed(3)
    tiles = torch.randint(0, 256, ((N + 15) // 16 * (K // 128), TILE_BYTES), dtype=torch.uint8, device=dev,
                          generator=g)
    tiles[:, 1024:1056].view(torch.int16).fill_(0x3C00)  # scales 2^-7 (bf16)
    tiles[:, 1056:] &= 15
    x = torch.randn(T, K, device=dev, generator=g).to(torch.bfloat16)
    y = torch.empty((T, N), dtype=torch.bfloat16, device=dev)
    err = torch.zeros(1, dtype=torch.int32, device=dev)
    for _ in range(args.warmup + args.reps):
        w4bf16_gemm(tiles.view(-1), x, N, out=y, err=err)
    torch.cuda.synchronize()
    flags = int(err.item())
    print(f"w4 GEMM T={T} N={N} K={K}: {args.warmup} + {args.reps} calls, device error word {flags}")
    return 0 if flags == 0 else 1


def run_layer_stage(args):
    """Runs --layer B,HIST: the attention half of one 8B-class decoder block (hidden 4096,
    Hq 32, Hkv 8, D 128) at HIST valid tokens through attn_decode_layer, --warmup + --reps
    times (no timing, no JSON line): the launch pattern of a profiler capture."""
    import torch

    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_15865_gb300.attention import Attention
    from paper_2607_15865_gb300.w4 import TILE_BYTES
    from synthetic.workloads import Shape
    bsz, hist = (int(v) for v in args.layer.split(","))
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    g = torch.Generator(device=dev).manual_seed(3)
    base = w.decode_shape(1)
    sh = Shape(f"layer_b{bsz}", bsz, base.n_q_heads, base.n_kv_heads, base.head_dim, base.max_len, base.rope_theta)
    hidden, qd, kd = 4096, sh.n_q_heads * sh.head_dim, sh.n_kv_heads * sh.head_dim

    def tiles(N, K):
        t = torch.randint(0, 256, ((N + 15) // 16 * (K // 128), TILE_BYTES), dtype=torch.uint8, device=dev, generator=g)
        t[:, 1024:1056].view(torch.int16).fill_(0x3C00)
        t[:, 1056:] &= 15
        return t.view(-1)

    def rnd(*shape):
        return (torch.randn(*shape, device=dev, generator=g) * 0.0884).to(torch.bfloat16)

    attn = Attention.for_shape(sh)
    tq, to = tiles(qd + 2 * kd, hidden), tiles(hidden, qd)
    kc = rnd(sh.batch, sh.n_kv_heads, sh.max_len, sh.head_dim)
    vc = rnd(sh.batch, sh.n_kv_heads, sh.max_len, sh.head_dim)
    x = torch.randn(bsz, hidden, device=dev, generator=g).to(torch.bfloat16)
    gamma = torch.ones(hidden, device=dev, dtype=torch.bfloat16)
    hl = torch.full((bsz,), hist, dtype=torch.int32, device=dev)
    for _ in range(args.warmup + args.reps):
        attn.decode_layer(x, gamma, 1e-6, tq, to, hl, kc, vc, weights_static=True)
    torch.cuda.synchronize()
    flags = attn.device_error()
    attn.close()
    print(f"decode block B{bsz} hist {hist}: {args.warmup} + {args.reps} calls, device error word {flags}")
    return 0 if flags == 0 else 1


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--cpu-rows", type=int, default=1536, help="prefill_kv rows in the oracle's timed sample")
    ap.add_argument("--ref-rows", type=int, default=48, help="prefill_kv rows per reference-arm step")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--sweep", action="store_true", help="time every configuration's stage instead (table to --sweep-out)")
    ap.add_argument("--sweep-out", default="sweep.json")
    ap.add_argument("--sweep-reps", type=int, default=20)
    ap.add_argument("--config-reps", type=int, default=15, help="calls per configuration row of the JSON line")
    ap.add_argument("--no-configs", action="store_true", help="leave the per-configuration rows out of the line")
    ap.add_argument("--stage", choices=tuple(STAGES), help="run only this stage (for profiler captures)")
    ap.add_argument("--reps", type=int, default=2)
    ap.add_argument("--hist", type=int)
    ap.add_argument("--chunk", type=int)
    ap.add_argument("--shape", choices=("long", "7b", "pkv512"), default="long",
                    help="with --stage: the long-context shape, the 7B-class prefill 512 or prefill_kv 512 over 1536")
    ap.add_argument("--w4", help="M,N,K: run only the W4BF16 GEMV of that shape (for profiler captures)")
    ap.add_argument("--layer", help="B,HIST: run only the W4BF16 decode block (for profiler captures)")
    ap.add_argument("--gemm", help="T,N,K: run only the W4BF16 GEMM of that shape (for profiler captures)")
    args = ap.parse_args()
    if args.stage:  # no timing in this mode
        return run_stage(args)
    if args.w4:
        return run_w4_stage(args)
    if args.layer:
        return run_layer_stage(args)
    if args.gemm:
        return run_gemm_stage(args)
    if args.warmup < 3:
        ap.error("--warmup must be at least 3")
    if args.impl == "reference":
        return run_reference(args)
    if args.sweep:
        return run_sweep(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
