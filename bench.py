"""Benchmark of the Nexus KV-cache splicing hot path on GB300.

One step = one pass of the whole path over the deep-context workload "c5"
(Qwen2.5-14B attention shape: 40 query / 8 KV heads, d = 128, 48 layers,
bf16, 16-token pages):

  1. splice: a 2048-token compiled block (anchor 0) inserted at depth 30000 of
     a 32768-token live cache, every layer, K reanchored by delta = 30000 and
     the 2768 displaced rows re-rotated by +2048 (one launch);
  2. re-prefill: causal self-attention of the 32768-token context, layer by
     layer (the R = 100 % end point of Eq. 2);
  3. suffix redecode: 64 queries over the 34816-token spliced cache, layer by
     layer, split-KV.

The printed metric is attention TFLOP/s over the whole step (algorithmic,
causal-visible flops 4 d Hq (R (T - R) + R (R + 1) / 2) per layer), with the
splice GB/s (8192 algorithmic bytes per moved token-layer) beside it. The fresh
Q/K/V of re-decoded tokens (projection + RoPE + cache write) is timed apart from
the step under "qkv_recompute" (2 x 5120 x 7168 flops per token), and the L0
warm arena (prefix match, fork, one boundary-page copy) under "l0_arena", and the
INT8 tool scan with its margin gate under "slb_route".

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Under torchrun every rank runs its own replica of the workload (the path
needs no exchange step); rank 0 prints the line with the max time over ranks.
"""
from __future__ import annotations

import argparse
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

METRIC = "suffix-redecode attention TFLOP/s + splice/rotate GB/s, % of GB300 roofline"
HQ, HKV, D, PAGE = 40, 8, 128, 16


def attn_flops(T: int, R: int, n_layers: int) -> float:
    return 4.0 * D * HQ * (R * (T - R) + R * (R + 1) / 2.0) * n_layers


def c5_config(L, n_past, Lb, depth, T, R, splits, world):
    return {"workload": f"c5 deep-context: {L} layers, n_past {n_past}, {Lb}-token block at "
                        f"{depth} (T={T}); re-prefill {n_past}x{n_past} causal + {R}-query "
                        f"split-KV suffix, 40/8 heads, d=128",
            "parallelism": f"replicas x{world}",
            "l2": "inputs exceed L2 (>30 GB touched per step); no flush"}


def max_over_ranks(x: float, dist, device) -> float:
    """Largest value of x over all ranks (identity without a process group)."""
    if dist is None:
        return float(x)
    import torch
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(flops_per_step_per_rank: float, world: int, ms_per_step: float) -> float:
    """Whole-job TFLOP/s: every rank runs its own replica of the step."""
    return world * flops_per_step_per_rank / (ms_per_step * 1e-3) / 1e12


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f), "measured"
    except OSError:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


# ------------------------------------------------------------------ clocks
class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = os.path.join("/tmp", f"nexus_clocks_{os.getpid()}.csv")

    def start(self):
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.f.close()
        sm, smax, power, reasons = [], [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    smax.append(float(parts[2]))
                    power.append(float(parts[3]))
                except ValueError:
                    continue
                for n, v in zip(names, parts[5:9]):
                    if v.lower().startswith("active"):
                        reasons.add(n)
        os.unlink(self.path)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        loaded = [s for s, p in zip(sm, power) if p > 0.5 * max(power)] or sm
        return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": max(smax),
                "power_w_max": max(power), "samples": len(sm), "reasons": sorted(reasons)}


# --------------------------------------------------------------- workload
class C5:
    """Device-resident c5 workload and the library calls of one step (also used
    with the c3 workload, whose cache keeps V token-innermost, for captures)."""

    def __init__(self, dev, n_layers=48, name="c5", prefill=True):
        import torch

        from paper_2608_20397_gb300 import nexus
        from paper_2608_20397_gb300.workloads import page_order, randn_bf16, workload

        self.torch, self.nexus = torch, nexus
        w = workload(name, n_layers=n_layers)
        self.w = w
        s = w.sessions[0]
        ins = s.inserts[0]
        L = w.n_layers
        self.L = L
        self.n_past, self.T = s.n_past, w.spliced_len(s)
        self.R_split = nexus.suffix_len(s.suffix_span, s.suffix_pct)
        self.depth, self.Lb = ins.depth, ins.length
        self.max_pages = -(-self.T // PAGE) + 1
        n_pages = -(-self.n_past // PAGE) + self.max_pages + 16
        self.pool = nexus.PagePool(n_pages, page_order(n_pages, w.seed, w.shuffle_pages))
        self.vt = w.v_transposed
        self.kp = torch.zeros((L, n_pages, HKV, PAGE, D), dtype=torch.bfloat16, device=dev)
        vshape = (L, n_pages, HKV, D, PAGE) if self.vt else (L, n_pages, HKV, PAGE, D)
        self.vp = torch.zeros(vshape, dtype=torch.bfloat16, device=dev)
        h_pt = np.full((2, self.max_pages), -1, np.int32)
        npg = -(-self.n_past // PAGE)
        h_pt[0, :npg] = self.pool.alloc(npg)
        # live cache straight into its pages, one layer at a time (setup only)
        pos = torch.arange(self.n_past, device=dev)
        pg = torch.as_tensor(h_pt[0], device=dev)[pos // PAGE].long()
        for l in range(L):
            k = randn_bf16((1, self.n_past, HKV, D), 500 + l, dev)
            v = randn_bf16((1, self.n_past, HKV, D), 600 + l, dev)
            self.kp[l, pg, :, pos % PAGE] = k[0]
            if self.vt:
                self.vp[l, pg, :, :, pos % PAGE] = v[0]
            else:
                self.vp[l, pg, :, pos % PAGE] = v[0]
        self.bk = randn_bf16((L, self.Lb, HKV, D), 700, dev)
        self.bv = randn_bf16((L, self.Lb, HKV, D), 701, dev)
        self.cache = nexus.kv_cache(self.kp, self.vp, n_pages, L, HKV, self.vt)
        self.blocks = [nexus.block(self.bk, self.bv, self.Lb, ins.base_pos, L, HKV)]
        new_pt, self.segs, _ = nexus.plan_splice(self.pool, h_pt[0], self.n_past, self.max_pages,
                                                 self.blocks, [(self.depth, 0)], 0, 1)
        h_pt[1] = new_pt
        self.h_pt = h_pt
        self.d_pt = torch.as_tensor(h_pt, device=dev)
        # the re-prefill's Q and O (16 GB each at 48 layers): only where they are used
        self.q_pre = randn_bf16((L, self.n_past, HQ, D), 800, dev) if prefill else None
        self.o_pre = torch.empty_like(self.q_pre) if prefill else None
        self.lse_pre = (torch.empty((L, self.n_past, HQ), dtype=torch.float32, device=dev)
                        if prefill else None)
        self.q_suf = randn_bf16((L, self.R_split, HQ, D), 900, dev)
        self.o_suf = torch.empty_like(self.q_suf)
        self.lse_suf = torch.empty((L, self.R_split, HQ), dtype=torch.float32, device=dev)
        self.ws_bytes, self.splits = nexus.attention_workspace_size([self.T], [self.R_split], HQ, HKV,
                                                                    1, 0)
        self.ws = torch.empty(max(16, self.ws_bytes), dtype=torch.uint8, device=dev)
        self.splice_rows = self.Lb + (self.n_past - self.depth)
        self.splice_bytes = 8192.0 * self.splice_rows * L
        self.flops_pre = attn_flops(self.n_past, self.n_past, L)
        self.flops_suf = attn_flops(self.T, self.R_split, L)
        # per layer: the re-prefill's plain grid plus the grid of its first tile
        # pairs (rows that see fewer than 128 keys); the suffix plus its merge
        self.launches_per_step = 1 + 2 * L + L * (2 if self.splits > 1 else 1)

    # library calls of one step; optional events bracket the splice and the re-prefill
    def step(self, stream, ev=None, q_pre=None, o_pre=None):
        nexus = self.nexus
        if ev is not None:
            ev[0].record(stream)
        nexus.splice_kv(self.cache, self.d_pt, None, 2, self.max_pages, self.blocks, self.segs, 0,
                        self.L, stream)
        if ev is not None:
            ev[1].record(stream)
        for l in range(self.L):
            nexus.reprefill(self.cache, self.d_pt, 2, self.max_pages, [self.n_past],
                            self.q_pre[l:l + 1] if q_pre is None else q_pre(l),
                            self.o_pre[l:l + 1] if o_pre is None else o_pre(l),
                            self.lse_pre[l:l + 1], HQ, l, l + 1, rows=[0], split_kv=1,
                            stream=stream)
        if ev is not None:
            ev[2].record(stream)
        for l in range(self.L):
            nexus.suffix_attention(self.cache, self.d_pt, 2, self.max_pages, [self.T],
                                   [self.R_split], self.q_suf[l:l + 1], self.o_suf[l:l + 1],
                                   self.lse_suf[l:l + 1], HQ, l, l + 1, rows=[1], split_kv=0,
                                   workspace=self.ws, workspace_bytes=self.ws_bytes, stream=stream)
        if ev is not None:
            ev[3].record(stream)


# ----------------------------------------------------------- cpu baseline
def oracle_sample_timing(q_rows, k, v, live_k, bk, n_rows_target_s=10.0, max_rows=64):
    """Times the fp64 oracle on a bounded sample of the same workload and
    returns (TFLOP/s, GB/s, description): attention rows of the re-prefill at
    the deep end of the context, and a splice of 64 block rows of one layer."""
    import oracle
    T = k.shape[0]
    flops, t_attn, rows_done = 0.0, 0.0, 0
    while rows_done < max_rows and t_attn < n_rows_target_s:
        r = min(4, max_rows - rows_done)
        pos = np.arange(T - r, T) - 4 * (rows_done // 4)
        t0 = time.perf_counter()
        oracle.attention(q_rows[rows_done:rows_done + r], k, v, pos, HQ // HKV)
        t_attn += time.perf_counter() - t0
        flops += sum(4.0 * D * HQ * (p + 1) for p in pos)
        rows_done += r
    t0 = time.perf_counter()
    oracle.splice_sequence(live_k, live_k, [(live_k.shape[1], bk, bk, 0)])
    t_spl = time.perf_counter() - t0
    spl_bytes = 8192.0 * bk.shape[1] * bk.shape[0]
    desc = (f"fp64 NumPy oracle: {rows_done} re-prefill query rows x {HQ} heads over ~{T} keys "
            f"(layer 0), and a {bk.shape[1]}-row block splice of one layer")
    return flops / t_attn / 1e12, spl_bytes / t_spl / 1e9, desc, t_attn + t_spl


def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count()


def run_reference(args):
    """Reference arm: the fp64 oracle as it stands, on the host cores, on a
    bounded sample of the c5 workload per step."""
    import torch

    from paper_2608_20397_gb300.workloads import randn_bf16
    f64 = lambda t: t.float().double().numpy()
    T = 32768
    k = f64(randn_bf16((T, HKV, D), 500, "cpu"))
    v = f64(randn_bf16((T, HKV, D), 600, "cpu"))
    q = f64(randn_bf16((64, HQ, D), 800, "cpu"))
    bk = f64(randn_bf16((1, 64, HKV, D), 700, "cpu"))
    live = f64(randn_bf16((1, 64, HKV, D), 501, "cpu"))
    vals, times, desc = [], [], ""
    for i in range(args.warmup + args.steps):
        t0 = time.perf_counter()
        tf, gbs, desc, _ = oracle_sample_timing(q, k, v, live, bk, n_rows_target_s=4.0, max_rows=16)
        dt = time.perf_counter() - t0
        if i >= args.warmup:
            vals.append(tf)
            times.append(dt)
    value = statistics.median(vals)
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "TFLOP/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * statistics.median(times), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": c5_config(48, 32768, 2048, 30000, 34816, 64, None, 1),
            "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": cpu_cores(),
                             "kind": "oracle", "sample": desc},
            "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------- main
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-qkv", action="store_true",
                    help="skip the separate timing of the suffix Q/K/V recompute")
    ap.add_argument("--no-arena", action="store_true",
                    help="skip the separate timing of the L0 warm arena")
    ap.add_argument("--no-slb", action="store_true",
                    help="skip the separate timing of the INT8 tool scan")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the separate timings of the workloads c1 .. c4")
    ap.add_argument("--layers", type=int, default=48, help="layers of the workload (48 = c5)")
    ap.add_argument("--profile", choices=["reprefill", "reprefill-softcap", "splice", "suffix",
                                          "qkv", "slb"],
                    default=None,
                    help="run only this kernel of the step (small case for ncu captures)")
    ap.add_argument("--workload", choices=["c5", "c3"], default="c5",
                    help="workload of --profile runs (c3: token-innermost V cache)")
    ap.add_argument("--tokens", type=int, default=0,
                    help="--profile qkv: re-decode this many last tokens of the spliced cache")
    ap.add_argument("--queries", type=int, default=1,
                    help="--profile slb: queries per launch (1..32)")
    args = ap.parse_args()

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if args.impl == "reference":
        if rank == 0:
            run_reference(args)
        return

    import torch
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)

    from paper_2608_20397_gb300 import nexus
    nexus.lib()
    if args.profile is None and args.workload != "c5":
        raise SystemExit("the timed step is the c5 workload; --workload only applies to --profile")
    wl = C5(dev, args.layers, args.workload,
            prefill=args.profile in (None, "reprefill", "reprefill-softcap"))
    stream = torch.cuda.current_stream()
    peaks, peak_kind = measured_peaks()

    def barrier():
        if dist is not None:
            dist.barrier()
        torch.cuda.synchronize()

    if args.profile:
        _profile_only(wl, args, stream)
        return

    for _ in range(args.warmup):
        wl.step(stream)
    st = nexus.device_status(stream)
    if st != nexus.OK:
        raise RuntimeError(f"device status after warm-up: {nexus.status_string(st)}")

    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(args.steps)]
    sampler = ClockSampler(dev.index)
    sampler.start()
    time.sleep(0.5)
    barrier()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for i in range(args.steps):
        wl.step(stream, evs[i])
    t_end.record(stream)
    barrier()
    clocks = sampler.stop()
    st = nexus.device_status(stream)
    if st != nexus.OK:
        raise RuntimeError(f"device status after timed steps: {nexus.status_string(st)}")
    total_ms = t_start.elapsed_time(t_end)
    splice_ms = statistics.mean(e[0].elapsed_time(e[1]) for e in evs)
    pre_ms = statistics.mean(e[1].elapsed_time(e[2]) for e in evs)
    suf_ms = statistics.mean(e[2].elapsed_time(e[3]) for e in evs)
    total_ms = max_over_ranks(total_ms, dist, dev)
    ms_per_step = total_ms / args.steps
    flops_step = wl.flops_pre + wl.flops_suf
    value = job_throughput(flops_step, world, ms_per_step)

    pre_launch_s = pre_ms * 1e-3 / wl.L
    achieved = (wl.flops_pre / wl.L) / pre_launch_s / 1e12
    peak_tc = peaks.get("bf16_tflops_sustained", peaks["bf16_tflops"])
    traffic = _profiled_traffic("attention_kernel")
    roofline = {"bound": "tensor", "kernel": "attention_kernel (re-prefill, one layer per launch)",
                "achieved": achieved, "peak": peak_tc, "unit": "TFLOP/s",
                "frac": achieved / peak_tc, "peak_kind": f"bf16 sustained, {peak_kind}",
                "traffic": traffic}
    splice_gbs = wl.splice_bytes / (splice_ms * 1e-3) / 1e9
    roofline_splice = {"bound": "hbm", "kernel": "splice_kernel", "achieved": splice_gbs,
                       "peak": peaks["hbm_gbs"], "unit": "GB/s",
                       "frac": splice_gbs / peaks["hbm_gbs"], "peak_kind": f"copy, {peak_kind}",
                       "frac_of_8tbs_spec": splice_gbs / 8000.0,
                       "traffic": _profiled_traffic("splice_kernel")}
    suf_tflops = wl.flops_suf / (suf_ms * 1e-3) / 1e12
    # The split-KV suffix sits near the ridge (about 320 flop per byte of K/V):
    # both fractions, per layer. Bytes: every key's K and V row of the layer
    # (8 KV heads x 128 x bf16, twice) plus Q read and O written.
    suf_bytes = wl.L * (wl.T * HKV * D * 2 * 2 + 2 * wl.R_split * HQ * D * 2)
    suf_gbs = suf_bytes / (suf_ms * 1e-3) / 1e9
    roofline_suffix = {"kernel": "attention_kernel + combine_kernel (split-KV suffix, "
                                 f"{wl.R_split} queries over {wl.T} keys, {wl.splits} splits)",
                       "achieved_tflops": suf_tflops, "frac_tensor": suf_tflops / peak_tc,
                       "achieved_gbs": suf_gbs, "frac_hbm": suf_gbs / peaks["hbm_gbs"],
                       "peak_kind": f"bf16 sustained / copy, {peak_kind}"}

    e2e = None
    if not args.no_e2e:
        e2e = _e2e(wl, stream, args, barrier, world, dist, dev)

    qkv = None
    if not args.no_qkv:
        qkv = _qkv_measure(wl, stream, peaks, peak_kind,
                           with_oracle=rank == 0 and world == 1 and not args.no_cpu_baseline)

    arena = None
    if not args.no_arena:
        arena = _arena_measure(wl, stream, peaks, peak_kind,
                               with_oracle=rank == 0 and world == 1 and not args.no_cpu_baseline)

    slb = None
    if not args.no_slb:
        slb = _slb_measure(wl, stream, peaks, peak_kind,
                           with_oracle=rank == 0 and world == 1 and not args.no_cpu_baseline)

    configs = None
    if not args.no_configs:
        configs = _configs_measure(dev, stream, peaks, peak_kind,
                                   with_oracle=rank == 0 and world == 1 and not args.no_cpu_baseline)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        f64 = lambda t: t.float().cpu().double().numpy()
        pos = torch.arange(wl.n_past, device=dev)
        pg = wl.d_pt[0][pos // PAGE].long()
        k0 = f64(wl.kp[0, pg, :, pos % PAGE])
        v0 = f64(wl.vp[0, pg, :, pos % PAGE])
        tf, gbs, desc, secs = oracle_sample_timing(f64(wl.q_pre[0, -64:]), k0, v0,
                                                   k0[None, :64], f64(wl.bk[:1, :64]))
        cpu = {"value": tf, "unit": "TFLOP/s", "cores": cpu_cores(), "kind": "oracle",
               "sample": desc, "splice_gbs": gbs, "seconds": secs}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic",
            "config": c5_config(wl.L, wl.n_past, wl.Lb, wl.depth, wl.T, wl.R_split, wl.splits,
                                world),
            "suffix_splits": wl.splits,
            "splice_gbs": splice_gbs, "splice_ms": splice_ms, "reprefill_ms": pre_ms,
            "suffix_ms": suf_ms, "suffix_tflops": suf_tflops, "roofline_suffix": roofline_suffix,
            "roofline": roofline, "roofline_splice": roofline_splice,
            "e2e": e2e, "cpu_baseline": cpu, "clocks": clocks, "qkv_recompute": qkv, "l0_arena": arena, "slb_route": slb,
            "configs": configs,
            "gpu_launches": wl.launches_per_step * args.steps,
        }
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()


def _profile_only(wl, args, stream):
    """W + K launches of one kernel of the step on the (reduced) workload,
    for ncu captures; prints the mean CUDA-event time per launch."""
    import torch
    nexus = wl.nexus
    if args.profile == "qkv":
        # Fresh Q, K, V of the re-decoded tokens of one layer: the 100 % suffix
        # of the spliced span (c3: 2192 tokens) or the whole context of the
        # re-prefill (c5: 32768 tokens).
        from paper_2608_20397_gb300.workloads import HIDDEN, qkv_weights, randn_bf16
        if args.tokens > 0:
            qkv_kv, qkv_n, qkv_row = wl.T, args.tokens, 1
        elif args.workload == "c3":
            qkv_kv, qkv_n, qkv_row = wl.T, wl.w.sessions[0].suffix_span, 1
        else:
            qkv_kv, qkv_n, qkv_row = wl.n_past, wl.n_past, 0
        dev = wl.kp.device
        qkv_x = randn_bf16((qkv_n, HIDDEN), 1000, dev)
        # three layers' weights in turn (220 MB, more than L2), as in the bench line
        qkv_wbs = [qkv_weights(HQ + 2 * HKV, HIDDEN, 1001 + i, dev) for i in range(3)]
        qkv_q = torch.empty((qkv_n, HQ, D), dtype=torch.bfloat16, device=dev)
        qkv_flops = 2.0 * qkv_n * HIDDEN * (HQ + 2 * HKV) * D
    launch_no = [0]

    if args.profile == "slb":
        # the 1M-tool registry of the bench's large tool scan, one query per launch
        dev = wl.kp.device
        g = torch.Generator(device=dev)
        g.manual_seed(12)
        slb_t = torch.randint(-127, 128, (1 << 20, 768), generator=g, device=dev,
                              dtype=torch.int32).to(torch.int8)
        slb_ts = torch.rand(1 << 20, generator=g, device=dev) * 0.01
        nq = max(1, min(32, args.queries))
        slb_q = torch.randint(-127, 128, (nq, 768), generator=g, device=dev,
                              dtype=torch.int32).to(torch.int8)
        slb_qs = torch.rand(nq, generator=g, device=dev) * 0.01
        slb_ws = torch.zeros(nexus.slb_workspace_size(1 << 20), dtype=torch.uint8, device=dev)
        slb_out = (torch.empty((nq, 2), dtype=torch.int32, device=dev),
                   torch.empty((nq, 2), dtype=torch.float32, device=dev),
                   torch.empty(nq, dtype=torch.int32, device=dev))

    def one():
        if args.profile == "slb":
            nexus.slb_route(slb_t, slb_ts, slb_q, slb_qs, *slb_out, slb_ws, stream=stream)
        elif args.profile == "qkv":
            qkv_w, qkv_b = qkv_wbs[launch_no[0] % 3]
            launch_no[0] += 1
            nexus.suffix_qkv(wl.cache, wl.d_pt, 2, wl.max_pages, [qkv_kv], [qkv_n], qkv_x, qkv_w,
                             qkv_b, qkv_q, layer=0, n_q_heads=HQ, rows=[qkv_row], stream=stream)
        elif args.profile == "splice":
            nexus.splice_kv(wl.cache, wl.d_pt, None, 2, wl.max_pages, wl.blocks, wl.segs, 0, wl.L,
                            stream)
        elif args.profile == "reprefill":
            nexus.reprefill(wl.cache, wl.d_pt, 2, wl.max_pages, [wl.n_past], wl.q_pre[:1],
                            wl.o_pre[:1], wl.lse_pre[:1], HQ, 0, 1, rows=[0], split_kv=1,
                            stream=stream)
        elif args.profile == "reprefill-softcap":
            nexus.suffix_attention_softcap(wl.cache, wl.d_pt, 2, wl.max_pages, [wl.n_past],
                                           [wl.n_past], wl.q_pre[:1], wl.o_pre[:1],
                                           wl.lse_pre[:1], HQ, 0, 1, rows=[0], split_kv=1,
                                           softcap=50.0, stream=stream)
        else:
            nexus.suffix_attention(wl.cache, wl.d_pt, 2, wl.max_pages, [wl.T], [wl.R_split],
                                   wl.q_suf[:1], wl.o_suf[:1], wl.lse_suf[:1], HQ, 0, 1, rows=[1],
                                   split_kv=0, workspace=wl.ws, workspace_bytes=wl.ws_bytes,
                                   stream=stream)

    for _ in range(args.warmup):
        one()
    torch.cuda.synchronize()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    # a fixed-length sleep holds the stream while the launches are enqueued, so
    # short launches are timed without the host's submission gaps
    torch.cuda._sleep(4_000_000)
    a.record(stream)
    for _ in range(args.steps):
        one()
    b.record(stream)
    torch.cuda.synchronize()
    st = nexus.device_status(stream)
    ms = a.elapsed_time(b) / args.steps
    if args.profile == "slb":
        gbs = (1 << 20) * 772.0 / (ms * 1e-3) / 1e9
        print(json.dumps({"profile": "slb", "tools": 1 << 20, "queries": args.queries,
                          "ms_per_launch": ms,
                          "rate": f"{gbs:.1f} GB/s", "status": nexus.status_string(st)}),
              flush=True)
        if st != nexus.OK:
            raise SystemExit(1)
        return
    if args.profile == "qkv":
        print(json.dumps({"profile": "qkv", "workload": args.workload, "tokens": qkv_n,
                          "ms_per_launch": ms,
                          "rate": f"{qkv_flops / (ms * 1e-3) / 1e12:.1f} TFLOP/s",
                          "status": nexus.status_string(st)}), flush=True)
        if st != nexus.OK:
            raise SystemExit(1)
        return
    rate = {"splice": f"{wl.splice_bytes / (ms * 1e-3) / 1e9:.1f} GB/s",
            "reprefill": f"{wl.flops_pre / wl.L / (ms * 1e-3) / 1e12:.1f} TFLOP/s",
            "reprefill-softcap": f"{wl.flops_pre / wl.L / (ms * 1e-3) / 1e12:.1f} TFLOP/s",
            "suffix": f"{wl.flops_suf / wl.L / (ms * 1e-3) / 1e12:.1f} TFLOP/s"}[args.profile]
    print(json.dumps({"profile": args.profile, "workload": args.workload, "layers": wl.L,
                      "ms_per_launch": ms, "rate": rate, "status": nexus.status_string(st)}),
          flush=True)
    if st != nexus.OK:
        raise SystemExit(1)


def _qkv_measure(wl, stream, peaks, peak_kind, with_oracle, warmup=3, reps=10):
    """Fresh Q, K, V of re-decoded tokens (one layer per launch), timed apart
    from the step: all 32768 tokens of the re-prefill (R = 100 %, Sec. III-C)
    and the 64-token suffix. Consecutive launches take the weights of different
    layers, three 73 MB matrices in turn (220 MB, more than L2), as a layer-by-
    layer re-decode does; the 64-token launch reads its weight from DRAM."""
    import torch

    from paper_2608_20397_gb300.workloads import HIDDEN, qkv_weights, randn_bf16
    nexus = wl.nexus
    dev = wl.kp.device
    n_heads = HQ + 2 * HKV
    wbs = [qkv_weights(n_heads, HIDDEN, 1001 + i, dev) for i in range(3)]
    w, b = wbs[0]
    x = randn_bf16((wl.n_past, HIDDEN), 1000, dev)
    q = torch.empty((wl.n_past, HQ, D), dtype=torch.bfloat16, device=dev)
    cases = {"reprefill": (wl.n_past, wl.n_past, 0), "suffix": (wl.T, wl.R_split, 1)}
    out = {"kernel": "qkv_kernel", "hidden": HIDDEN, "heads": f"{HQ} q + {HKV} k + {HKV} v",
           "weights": "three layers' weights in turn (220 MB > L2)"}
    for name, (kv, n, row) in cases.items():
        def one(l):
            wl_, bl_ = wbs[l % 3]
            nexus.suffix_qkv(wl.cache, wl.d_pt, 2, wl.max_pages, [kv], [n], x[:n], wl_, bl_,
                             q[:n], layer=l % wl.L, n_q_heads=HQ, rows=[row], stream=stream)
        for i in range(warmup):
            one(i)
        a = torch.cuda.Event(enable_timing=True)
        e = torch.cuda.Event(enable_timing=True)
        # a fixed-length sleep holds the stream while the launches are enqueued,
        # so short launches are timed without the host's submission gaps
        torch.cuda.synchronize()
        torch.cuda._sleep(4_000_000)
        a.record(stream)
        t0 = time.perf_counter()
        for i in range(reps):
            one(i)
        host_us = (time.perf_counter() - t0) / reps * 1e6
        e.record(stream)
        torch.cuda.synchronize()
        ms = a.elapsed_time(e) / reps
        flops = 2.0 * n * HIDDEN * n_heads * D
        out[name] = {"tokens": n, "ms_per_launch": ms, "tflops": flops / (ms * 1e-3) / 1e12,
                     "host_us_per_call": host_us}
    st = nexus.device_status(stream)
    if st != nexus.OK:
        raise RuntimeError(f"device status after the Q/K/V timing: {nexus.status_string(st)}")
    achieved = out["reprefill"]["tflops"]
    out["roofline"] = {"bound": "tensor", "kernel": "qkv_kernel (32768 tokens, one layer)",
                       "achieved": achieved, "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
                       "frac": achieved / peaks["bf16_tflops"],
                       "peak_kind": f"bf16 burst (timed alone), {peak_kind}",
                       "traffic": _profiled_traffic("qkv_kernel")}
    if with_oracle:
        import oracle
        n = 64
        xs = x[:n].float().cpu().double().numpy()
        wf = w.float().cpu().double().numpy()
        bf = b.double().cpu().numpy()
        t0 = time.perf_counter()
        oracle.qkv_recompute(xs, wf, bf, np.arange(n), HQ, HKV)
        dt = time.perf_counter() - t0
        out["cpu_baseline"] = {"value": 2.0 * n * HIDDEN * n_heads * D / dt / 1e12,
                               "unit": "TFLOP/s", "cores": cpu_cores(), "kind": "oracle",
                               "sample": f"fp64 NumPy oracle: {n} tokens x {HIDDEN} hidden -> "
                                         f"{n_heads * D} features, with RoPE", "seconds": dt}
    return out


def _arena_measure(wl, stream, peaks, peak_kind, with_oracle, n_slots=32, system_len=8192,
                   tail_len=1024, n_requests=200):
    """The L0 warm arena (Sec. V-D), timed apart from the step on a cache of the
    c5 model shape (48 layers, 8 KV heads): 32 slots holding a shared
    8192-token system prompt plus a 1024-token tail each; every request shares
    the prompt and part of one tail, so it forks 8192 + k warm tokens (k random)
    and copies one boundary page of all 48 layers. Also the warm-hit rate of
    the arena on a seeded stream of agent requests (context: it depends wholly on
    the stream)."""
    import torch

    from paper_2608_20397_gb300.workloads import agent_requests
    nexus = wl.nexus
    dev = wl.kp.device
    L = wl.L
    r = np.random.default_rng(77)
    sys_pages = system_len // PAGE
    tail_pages = tail_len // PAGE
    n_pages = sys_pages + n_slots * tail_pages + 64
    kp = torch.zeros((L, n_pages, HKV, PAGE, D), dtype=torch.bfloat16, device=dev)
    vp = torch.zeros_like(kp)
    cache = nexus.kv_cache(kp, vp, n_pages, L, HKV)
    pool = nexus.PagePool(n_pages)
    arena = nexus.WarmArena(n_slots, system_len + tail_len)
    system = [int(t) for t in r.integers(0, 32000, system_len)]
    sys_pt = pool.alloc(sys_pages)
    tails = []
    for s in range(n_slots):
        tail = [int(t) for t in r.integers(0, 32000, tail_len)]
        tails.append(tail)
        pt = np.concatenate([sys_pt, pool.alloc(tail_pages)]).astype(np.int32)
        pool.retain(sys_pt)
        arena.store(pool, system + tail, pt)
        pool.free(pt)
    pool.free(sys_pt)            # the slots alone hold the pages now
    reqs = []
    for i in range(n_requests + 10):
        j = int(r.integers(0, n_slots))
        k = int(r.integers(1, tail_len))
        q = system + tails[j][:k] + [int(t) for t in r.integers(32000, 33000, 64)]
        reqs.append((np.asarray(q, dtype=np.int32), system_len + k))
    # one request at a time, as a server sees it: match, fork, boundary copy, done
    t_match, t_fork, t_e2e = [], [], []
    for i, (q, m_want) in enumerate(reqs):
        stream.synchronize()
        t0 = time.perf_counter()
        slot, m = arena.match(q)
        t1 = time.perf_counter()
        pt, src, dst = arena.fork(pool, slot, m, -(-len(q) // PAGE))
        t2 = time.perf_counter()
        if len(src):
            nexus.copy_pages(cache, src, dst, 0, L, stream)
        stream.synchronize()
        t3 = time.perf_counter()
        assert m >= m_want
        pool.free(pt)
        if i >= 10:
            t_match.append(t1 - t0)
            t_fork.append(t2 - t1)
            t_e2e.append(t3 - t0)
    # the boundary copies alone: a batch enqueued while the stream is held busy
    # by a fixed-length sleep, so the events see no host gaps
    t_copy = []
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    for rep in range(5):
        plans = []
        for q, _ in reqs[rep * 40:(rep + 1) * 40]:
            slot, m = arena.match(q)
            plans.append(arena.fork(pool, slot, m, -(-len(q) // PAGE)))
        copies = [(src, dst) for _, src, dst in plans if len(src)]
        torch.cuda._sleep(4_000_000)
        ev[0].record(stream)
        for src, dst in copies:
            nexus.copy_pages(cache, src, dst, 0, L, stream)
        ev[1].record(stream)
        ev[1].synchronize()
        if rep > 0 and copies:
            t_copy.append(ev[0].elapsed_time(ev[1]) * 1e-3 / len(copies))
        for pt, _, _ in plans:
            pool.free(pt)
    st = nexus.device_status(stream)
    if st != nexus.OK:
        raise RuntimeError(f"device status after the arena timing: {nexus.status_string(st)}")
    p50 = lambda xs: float(np.median(xs)) * 1e6
    page_bytes = 2.0 * 2 * L * HKV * PAGE * D * 2     # K and V of one page, read + written
    copy_us = p50(t_copy)
    out = {"slots": n_slots, "layers": L,
           "setup": f"{n_slots} slots: a shared {system_len}-token prompt + a {tail_len}-token "
                    f"tail each; requests fork {system_len} + U[1, {tail_len}) warm tokens",
           "match_us_p50": p50(t_match), "fork_host_us_p50": p50(t_fork),
           "copy_us_mean": copy_us, "fork_e2e_us_p50": p50(t_e2e),
           "timing": "match / fork / e2e: wall clock through the Python binding, one request "
                     "at a time (e2e ends when the copy has run); copy: CUDA events over 40 "
                     "back-to-back boundary copies",
           "roofline": {"bound": "hbm", "kernel": "page_copy_kernel (one boundary page, "
                                                 f"{L} layers, K and V)",
                        "achieved": page_bytes / (copy_us * 1e-6) / 1e9, "peak": peaks["hbm_gbs"],
                        "unit": "GB/s", "frac": page_bytes / (copy_us * 1e-6) / 1e9 / peaks["hbm_gbs"],
                        "peak_kind": f"copy, {peak_kind}", "traffic": None,
                        "note": "6.3 MB per launch: too small to reach the HBM bound"}}
    arena.close(pool)
    del kp, vp
    # warm-hit rate on a seeded agent stream (host only)
    pool2 = nexus.PagePool(1 << 16)
    ar2 = nexus.WarmArena(n_slots, 1 << 14)
    hits = reused = total = 0
    for q in agent_requests(11, 2000, n_agents=48, sys_len=600, vocab=32000):
        slot, m = ar2.match(q)
        npg = -(-len(q) // PAGE)
        pre = np.zeros(0, np.int32)
        if slot >= 0:
            pre, _, _ = ar2.fork(pool2, slot, m, npg)
            hits += m > 0
        pt = np.concatenate([pre, pool2.alloc(npg - len(pre))]).astype(np.int32)
        ar2.store(pool2, q, pt)
        pool2.free(pt)
        reused += m
        total += len(q)
    ar2.close(pool2)
    out["hit_rate"] = hits / 2000.0
    out["token_reuse"] = reused / total
    out["hit_stream"] = "2000 seeded requests of 48 agents sharing a 600-token prompt"
    if with_oracle:
        import oracle
        model = oracle.WarmArenaModel(n_slots, system_len + tail_len)
        for s in range(n_slots):
            z = np.zeros((1, system_len + tail_len, 1, 1))
            model.store(system + tails[s], z, z)
        q = system + tails[0][:500] + [32001]
        t0 = time.perf_counter()
        reps = 3
        for _ in range(reps):
            model.match(q)
        dt = (time.perf_counter() - t0) / reps
        out["cpu_baseline"] = {"value": dt * 1e6, "unit": "us per match", "cores": 1,
                               "kind": "oracle",
                               "sample": f"plain-Python model: one {len(q)}-token query against "
                                         f"the same {n_slots} slots"}
    return out


def _slb_measure(wl, stream, peaks, peak_kind, with_oracle, reps=200):
    """The INT8 tool scan and margin gate (Sec. IV-A), timed apart from the step:
    (a) the paper's size, 250 tools x 768 dims, one query: the kernel alone
    (CUDA events over back-to-back launches enqueued behind a fixed sleep) and a
    whole routing call from a host embedding (quantise, copy in, scan, copy the
    decision out, P50); (b) a registry of 1M tools (768 MB of codes, larger than
    L2) at 1, 8 and 32 queries per launch; the single query, which only streams
    the codes, against the HBM roofline."""
    import torch

    from paper_2608_20397_gb300.workloads import tool_queries, tool_registry
    nexus = wl.nexus
    dev = wl.kp.device
    x = tool_registry(250)
    q, _ = tool_queries(x, reps + 10)
    tc, ts = nexus.slb_quantize(x)
    d_tc = torch.as_tensor(tc, device=dev)
    d_ts = torch.as_tensor(ts, device=dev)
    ws = torch.zeros(nexus.slb_workspace_size(250), dtype=torch.uint8, device=dev)
    top_idx = torch.empty((32, 2), dtype=torch.int32, device=dev)
    top_score = torch.empty((32, 2), dtype=torch.float32, device=dev)
    route = torch.empty(32, dtype=torch.int32, device=dev)
    h_qc = torch.empty((1, 768), dtype=torch.int8, pin_memory=True)
    h_qs = torch.empty(1, dtype=torch.float32, pin_memory=True)
    h_out = torch.empty(3, dtype=torch.int32, pin_memory=True)
    d_qc = torch.empty((1, 768), dtype=torch.int8, device=dev)
    d_qs = torch.empty(1, dtype=torch.float32, device=dev)
    t_e2e = []
    for i in range(reps + 10):
        stream.synchronize()
        t0 = time.perf_counter()
        qc, qs = nexus.slb_quantize(q[i:i + 1])
        h_qc.numpy()[:] = qc
        h_qs.numpy()[:] = qs
        d_qc.copy_(h_qc, non_blocking=True)
        d_qs.copy_(h_qs, non_blocking=True)
        nexus.slb_route(d_tc, d_ts, d_qc, d_qs, top_idx[:1], top_score[:1], route[:1], ws,
                        stream=stream)
        h_out[:2].copy_(top_idx[0], non_blocking=True)
        h_out[2:].copy_(route[:1], non_blocking=True)
        stream.synchronize()
        if i >= 10:
            t_e2e.append(time.perf_counter() - t0)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    def kernel_us(tools, scales, queries, qscales, n_launch, w):
        torch.cuda._sleep(4_000_000)
        ev[0].record(stream)
        for _ in range(n_launch):
            nexus.slb_route(tools, scales, queries, qscales, top_idx[:queries.shape[0]],
                            top_score[:queries.shape[0]], route[:queries.shape[0]], w,
                            stream=stream)
        ev[1].record(stream)
        ev[1].synchronize()
        return ev[0].elapsed_time(ev[1]) * 1e3 / n_launch
    kernel_us(d_tc, d_ts, d_qc, d_qs, 10, ws)
    small_us = float(np.median([kernel_us(d_tc, d_ts, d_qc, d_qs, 50, ws) for _ in range(5)]))
    # 1M tools: codes and scales drawn on the device (the scan's time does not
    # depend on the values)
    n_big, dim = 1 << 20, 768
    g = torch.Generator(device=dev)
    g.manual_seed(12)
    big = torch.randint(-127, 128, (n_big, dim), generator=g, device=dev, dtype=torch.int32).to(torch.int8)
    big_s = torch.rand(n_big, generator=g, device=dev) * 0.01
    bq = torch.randint(-127, 128, (32, dim), generator=g, device=dev, dtype=torch.int32).to(torch.int8)
    bqs = torch.rand(32, generator=g, device=dev) * 0.01
    ws_big = torch.zeros(nexus.slb_workspace_size(n_big), dtype=torch.uint8, device=dev)
    big_bytes = n_big * (dim + 4.0)
    by_batch = {}
    for nb in (1, 8, 32):
        kernel_us(big, big_s, bq[:nb], bqs[:nb], 2, ws_big)
        us = float(np.median([kernel_us(big, big_s, bq[:nb], bqs[:nb], 5, ws_big)
                              for _ in range(3)]))
        by_batch[nb] = {"kernel_us": us, "gbs": big_bytes / (us * 1e-6) / 1e9,
                        "queries_per_s": nb / (us * 1e-6)}
    one_us = by_batch[1]["kernel_us"]
    st = nexus.device_status(stream)
    if st != nexus.OK:
        raise RuntimeError(f"device status after the tool-scan timing: {nexus.status_string(st)}")
    gbs = big_bytes / (one_us * 1e-6) / 1e9
    out = {"kernel": "slb_kernel",
           "paper_size": {"tools": 250, "dim": 768, "queries": 1, "kernel_us": small_us,
                          "route_e2e_us_p50": float(np.median(t_e2e)) * 1e6,
                          "e2e": "host embedding -> quantise -> copy in -> scan + gate -> "
                                 "decision copied out, through the Python binding"},
           "large": {"tools": n_big, "dim": dim, "by_batch": by_batch,
                     "note": "8 and 32 queries per launch: exact bf16 tensor-core scan "
                             "(slb_tc_kernel), flat in the batch size at ~2.5 TB/s"},
           "roofline": {"bound": "hbm", "kernel": "slb_stream_kernel (1M x 768 codes, 1 query)",
                        "achieved": gbs, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                        "frac": gbs / peaks["hbm_gbs"], "peak_kind": f"copy, {peak_kind}",
                        "traffic": _profiled_traffic("slb_stream_kernel")}}
    del big, ws_big
    if with_oracle:
        import oracle
        oc, os_ = oracle.slb_quantize(x)
        qc, qs = oracle.slb_quantize(q[:20])
        t0 = time.perf_counter()
        for i in range(20):
            oracle.slb_route(qc[i:i + 1], qs[i:i + 1], oc, os_)
        dt = (time.perf_counter() - t0) / 20
        out["cpu_baseline"] = {"value": dt * 1e6, "unit": "us per query", "cores": 1,
                               "kind": "oracle",
                               "sample": "NumPy oracle: one query against 250 x 768 codes"}
    return out


# ---------------------------------------------------- configs c1 .. c4
class ConfigCase:
    """One of the workloads c1 .. c4 resident on the device: every session's live
    rows in a paged pool (N(0, 1) bf16, pages handed out in the workload's
    order), its compiled blocks, the planned splice (page-table rows 2 s / 2 s + 1
    before / after the splice) and the suffix queries of each redecode fraction."""

    def __init__(self, name, dev):
        import torch

        from paper_2608_20397_gb300 import nexus
        from paper_2608_20397_gb300.workloads import page_order, randn_bf16, workload

        self.torch, self.nexus = torch, nexus
        w = workload(name)
        self.w, self.name, self.L, self.vt = w, name, w.n_layers, w.v_transposed
        S = len(w.sessions)
        self.kv = [w.spliced_len(s) for s in w.sessions]
        pages = sum(-(-s.n_past // PAGE) + -(-t // PAGE) + 1 for s, t in zip(w.sessions, self.kv))
        self.n_pages = pages + 64
        self.max_pages = max(-(-t // PAGE) for t in self.kv) + 1
        self.pool = nexus.PagePool(self.n_pages, page_order(self.n_pages, w.seed, w.shuffle_pages))
        g = torch.Generator(device=dev)
        g.manual_seed(9000 + w.seed)
        # Every slot of the pool holds N(0, 1) bf16: the live rows are whatever
        # the pages hold (the timing does not depend on which values they are).
        self.kp = torch.empty((self.L, self.n_pages, HKV, PAGE, D), dtype=torch.bfloat16, device=dev)
        vshape = (self.L, self.n_pages, HKV, D, PAGE) if self.vt else self.kp.shape
        self.vp = torch.empty(vshape, dtype=torch.bfloat16, device=dev)
        for l in range(self.L):
            self.kp[l].normal_(generator=g)
            self.vp[l].normal_(generator=g)
        self.cache = nexus.kv_cache(self.kp, self.vp, self.n_pages, self.L, HKV, self.vt,
                                    rope_theta=w.rope_theta)
        h_pt = np.full((2 * S, self.max_pages), -1, np.int32)
        self.blocks, self.segs, self._blk = [], [], []
        for si, s in enumerate(w.sessions):
            npg = -(-s.n_past // PAGE)
            h_pt[2 * si, :npg] = self.pool.alloc(npg)
            base = len(self.blocks)
            for j, ins in enumerate(s.inserts):
                bk = randn_bf16((self.L, ins.length, HKV, D), 20000 + 10 * si + 2 * j, dev)
                bv = randn_bf16((self.L, ins.length, HKV, D), 20001 + 10 * si + 2 * j, dev)
                self._blk += [bk, bv]
                self.blocks.append(nexus.block(bk, bv, ins.length, ins.base_pos, self.L, HKV,
                                               rope_theta=w.rope_theta))
            new_pt, segs, _ = nexus.plan_splice(
                self.pool, h_pt[2 * si], s.n_past, self.max_pages, self.blocks,
                [(ins.depth, base + j) for j, ins in enumerate(s.inserts)], 2 * si, 2 * si + 1,
                seg_capacity=4 * len(s.inserts) + 4)
            h_pt[2 * si + 1] = new_pt
            self.segs += segs
        self.h_pt = h_pt
        self.d_pt = torch.as_tensor(h_pt, device=dev)
        self.n_rows = 2 * S
        # every segment moves its rows' K and V: 8192 bytes per row and layer
        self.moved_rows = sum(int(sg.n_tokens) for sg in self.segs)
        self.splice_bytes = 8192.0 * self.moved_rows * self.L
        pcts = w.suffix_pcts or (w.sessions[0].suffix_pct,)
        self.q_len = {p: [nexus.suffix_len(s.suffix_span, p) for s in w.sessions] for p in pcts}

    def splice(self, stream):
        self.nexus.splice_kv(self.cache, self.d_pt, None, self.n_rows, self.max_pages, self.blocks,
                             self.segs, 0, self.L, stream)

    def flops(self, pct):
        return sum(attn_flops(T, R, self.L) for T, R in zip(self.kv, self.q_len[pct]))


def _time_back_to_back(fn, stream, warmup, reps):
    """Mean CUDA-event time (ms) of `reps` back-to-back calls, enqueued behind a
    fixed-length sleep so that short launches are timed without host gaps."""
    import torch
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    torch.cuda._sleep(4_000_000)
    a.record(stream)
    for _ in range(reps):
        fn()
    b.record(stream)
    torch.cuda.synchronize()
    return a.elapsed_time(b) / reps


def _oracle_config_sample(T, R, budget_s=1.0):
    """The fp64 oracle on a bounded sample of a config's suffix attention (one
    layer, rows from the deep end of the suffix, N(0, 1) inputs) and of its
    splice (a 64-row block into a 64-row cache, one layer). Returns (attention
    TFLOP/s, splice GB/s, description)."""
    import oracle
    from paper_2608_20397_gb300.workloads import randn_bf16
    f64 = lambda t: t.float().double().numpy()
    rows_max = min(R, 64)
    q = f64(randn_bf16((rows_max, HQ, D), 31, "cpu"))
    k = f64(randn_bf16((T, HKV, D), 32, "cpu"))
    v = f64(randn_bf16((T, HKV, D), 33, "cpu"))
    flops, spent, done = 0.0, 0.0, 0
    while done < rows_max and (spent < budget_s or done == 0):
        r = min(4, rows_max - done)
        pos = np.arange(T - done - r, T - done)
        t0 = time.perf_counter()
        oracle.attention(q[done:done + r], k, v, pos, HQ // HKV)
        spent += time.perf_counter() - t0
        flops += sum(4.0 * D * HQ * (p + 1) for p in pos)
        done += r
    live = f64(randn_bf16((1, 64, HKV, D), 34, "cpu"))
    blk = f64(randn_bf16((1, 64, HKV, D), 35, "cpu"))
    t0 = time.perf_counter()
    oracle.splice_sequence(live, live, [(32, blk, blk, 0)])
    t_spl = time.perf_counter() - t0
    desc = (f"fp64 NumPy oracle: {done} suffix rows x {HQ} heads over up to {T} keys (one layer), "
            f"and a 64-row block splice into a 64-row cache (one layer)")
    return flops / spent / 1e12, 8192.0 * 96 / t_spl / 1e9, desc


def _configs_measure(dev, stream, peaks, peak_kind, with_oracle, warmup=3, reps=10):
    """c1 .. c4 timed one after another, apart from the c5 step: the splice of
    each (hot, and for the single-layer c1 / c2, whose moved rows fit in L2,
    also with a 512 MB scratch write between launches) and its suffix attention
    at every redecode fraction the config names (one launch per layer), each
    against its roofline, with the fp64 oracle on a bounded sample beside it."""
    import torch
    nexus = None
    peak_tc = peaks["bf16_tflops"]
    out = {}
    for name in ("c1", "c2", "c3", "c4"):
        case = ConfigCase(name, dev)
        nexus = case.nexus
        w = case.w
        line = {"layers": case.L, "sessions": len(w.sessions),
                "v_layout": "token-innermost" if case.vt else "row-major",
                "pages": "shuffled" if w.shuffle_pages else "in order",
                "kv_len": case.kv if len(case.kv) <= 2 else
                {"min": min(case.kv), "max": max(case.kv), "sum": sum(case.kv)}}
        ms = _time_back_to_back(lambda: case.splice(stream), stream, warmup, reps)
        gbs = case.splice_bytes / (ms * 1e-3) / 1e9
        spl = {"moved_rows_per_layer": case.moved_rows, "bytes": case.splice_bytes,
               "ms": ms, "gbs": gbs, "frac": gbs / peaks["hbm_gbs"],
               "bound": "hbm", "peak": peaks["hbm_gbs"], "peak_kind": f"copy, {peak_kind}",
               "timing": "back to back (moved rows L2-resident where they fit)"}
        if case.L == 1:
            flush = torch.empty(512 << 20, dtype=torch.uint8, device=dev)
            evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                   for _ in range(reps)]
            for i in range(warmup + reps):
                flush.fill_(i & 255)
                if i >= warmup:
                    evs[i - warmup][0].record(stream)
                case.splice(stream)
                if i >= warmup:
                    evs[i - warmup][1].record(stream)
            torch.cuda.synchronize()
            msf = statistics.mean(a.elapsed_time(b) for a, b in evs)
            gf = case.splice_bytes / (msf * 1e-3) / 1e9
            spl.update({"ms_l2_flushed": msf, "gbs_l2_flushed": gf,
                        "frac_l2_flushed": gf / peaks["hbm_gbs"],
                        "flush": "512 MB scratch write before each timed launch (events per launch)"})
            del flush
        line["splice"] = spl
        case.splice(stream)
        torch.cuda.synchronize()
        sufs = []
        for pct, ql in case.q_len.items():
            n_tok = sum(ql)
            q = torch.empty((case.L, n_tok, HQ, D), dtype=torch.bfloat16, device=dev).normal_()
            o = torch.empty_like(q)
            lse = torch.empty((case.L, n_tok, HQ), dtype=torch.float32, device=dev)
            wsb, splits = nexus.attention_workspace_size(case.kv, ql, HQ, HKV, 1, 0)
            ws = torch.empty(max(16, wsb), dtype=torch.uint8, device=dev)
            rows = [2 * i + 1 for i in range(len(w.sessions))]

            def run():
                for l in range(case.L):
                    nexus.suffix_attention(case.cache, case.d_pt, case.n_rows, case.max_pages,
                                           case.kv, ql, q[l:l + 1], o[l:l + 1], lse[l:l + 1], HQ,
                                           l, l + 1, rows=rows, split_kv=0, workspace=ws,
                                           workspace_bytes=wsb, stream=stream)
            ms = _time_back_to_back(run, stream, warmup, reps)
            tf = case.flops(pct) / (ms * 1e-3) / 1e12
            sufs.append({"pct": pct, "q_len": ql if len(ql) <= 2 else {"sum": n_tok},
                         "splits": splits, "ms": ms, "ms_per_layer": ms / case.L,
                         "tflops": tf, "frac": tf / peak_tc, "bound": "tensor",
                         "peak": peak_tc, "peak_kind": f"bf16 burst (timed alone), {peak_kind}"})
            del q, o, lse, ws
        line["suffix_attention"] = sufs
        st = nexus.device_status(stream)
        if st != nexus.OK:
            raise RuntimeError(f"device status after config {name}: {nexus.status_string(st)}")
        if with_oracle:
            T = max(case.kv)
            R = max(max(v) for v in case.q_len.values())
            tf, g, desc = _oracle_config_sample(T, R)
            line["cpu_baseline"] = {"value": tf, "unit": "TFLOP/s", "cores": cpu_cores(),
                                    "kind": "oracle", "sample": desc, "splice_gbs": g}
        out[name] = line
        del case
        torch.cuda.empty_cache()
    return out


def _profiled_traffic(kernel: str):
    """DRAM bytes (read + write) per launch from the committed ncu summary, or
    None when there is none or the kernel source changed since the capture."""
    import hashlib
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            entry = json.load(f).get(kernel)
        if not entry:
            return None
        with open(os.path.join(ROOT, entry["source"]), "rb") as f:
            if hashlib.sha256(f.read()).hexdigest() != entry["source_sha256"]:
                return None
        return entry["bytes_per_launch"]
    except (OSError, ValueError, KeyError):
        return None


def _huge_page_fraction(tensors):
    """Fraction of the bytes of the mappings that hold these host tensors that
    the kernel backs with transparent huge pages (Linux /proc/self/smaps), or
    None where that cannot be read. Copies from page-locked memory on scattered
    base pages run several times slower, so this explains a slow e2e line."""
    spans = [(t.data_ptr(), t.data_ptr() + t.numel() * t.element_size()) for t in tensors]
    try:
        size = huge = 0
        cur = None
        with open("/proc/self/smaps") as f:
            for line in f:
                head = line.split()[0]
                if "-" in head and not head.endswith(":"):
                    lo, hi = (int(x, 16) for x in head.split("-"))
                    cur = any(a < hi and lo < b for a, b in spans)
                elif cur and head == "Size:":
                    size += int(line.split()[1])
                elif cur and head == "AnonHugePages:":
                    huge += int(line.split()[1])
        return huge / size if size else None
    except (OSError, ValueError):
        return None


def _e2e(wl, stream, args, barrier, world, dist, dev):
    """The same step through the C ABI with host buffers: every step copies the
    block K/V and every layer's Q in from pinned host memory and reads every
    layer's O back, inside the timed region. Copies run on their own streams,
    double-buffered per layer, so they overlap the attention of other layers."""
    import torch
    L = wl.L
    nexus = wl.nexus
    # Host buffers in the library's page-locked staging memory (nexus_host_alloc,
    # huge pages where the request is large): every layer's Q in one region, the
    # two O buffers in another, the rest in a third.
    # The block K/V and the suffix's Q and O share one region, so that they sit in
    # huge pages too (each alone is under the size that gets them).
    host = lambda shape, dtype=torch.bfloat16: nexus.host_empty(shape, dtype)
    bf16 = torch.bfloat16
    h_bk, h_bv, h_qs, h_os = nexus.host_empty_group(
        [(wl.bk.shape, bf16), (wl.bv.shape, bf16), (wl.q_suf.shape, bf16), (wl.o_suf.shape, bf16)])
    h_bk.copy_(wl.bk)
    h_bv.copy_(wl.bv)
    h_qall = host(wl.q_pre.shape)
    h_q = [h_qall[l] for l in range(L)]
    h_oall = host((2,) + tuple(wl.o_pre.shape[1:]))
    h_o = [h_oall[0], h_oall[1]]
    h_qall.copy_(wl.q_pre)
    h_qs.copy_(wl.q_suf)
    qbuf = [torch.empty_like(wl.q_pre[:1]) for _ in range(2)]
    obuf = [torch.empty_like(wl.o_pre[:1]) for _ in range(2)]
    s_in = torch.cuda.Stream(device=dev)
    s_out = torch.cuda.Stream(device=dev)
    h2d = (h_bk.numel() + h_bv.numel() + sum(x.numel() for x in h_q) + h_qs.numel()) * 2
    d2h = (L * h_o[0].numel() + h_os.numel()) * 2
    ev = lambda: torch.cuda.Event()

    def one():
        # Layer 0's block rows and queries go first; the other layers' block rows
        # follow and are spliced while layer 0's attention runs.
        e_blk0, e_blk = ev(), ev()
        with torch.cuda.stream(s_in):
            wl.bk[:1].copy_(h_bk[:1], non_blocking=True)
            wl.bv[:1].copy_(h_bv[:1], non_blocking=True)
            e_blk0.record(s_in)
        stream.wait_event(e_blk0)
        nexus.splice_kv(wl.cache, wl.d_pt, wl.h_pt, 2, wl.max_pages, wl.blocks, wl.segs, 0, 1,
                        stream)
        e_in = [None] * L
        e_done = [None] * L
        e_out = [None] * L
        for l in range(L):
            b = l & 1
            with torch.cuda.stream(s_in):
                if l >= 2:
                    s_in.wait_event(e_done[l - 2])     # attention of layer l-2 read qbuf[b]
                qbuf[b][0].copy_(h_q[l], non_blocking=True)
                e_in[l] = ev()
                e_in[l].record(s_in)
                if l == 0:
                    wl.bk[1:].copy_(h_bk[1:], non_blocking=True)
                    wl.bv[1:].copy_(h_bv[1:], non_blocking=True)
                    wl.q_suf.copy_(h_qs, non_blocking=True)
                    e_blk.record(s_in)
            if l == 1:
                stream.wait_event(e_blk)
                nexus.splice_kv(wl.cache, wl.d_pt, wl.h_pt, 2, wl.max_pages, wl.blocks, wl.segs,
                                1, L, stream)
            stream.wait_event(e_in[l])
            if l >= 2:
                stream.wait_event(e_out[l - 2])        # O of layer l-2 left obuf[b]
            nexus.reprefill(wl.cache, wl.d_pt, 2, wl.max_pages, [wl.n_past], qbuf[b], obuf[b],
                            wl.lse_pre[l:l + 1], HQ, l, l + 1, rows=[0], split_kv=1,
                            stream=stream)
            e_done[l] = ev()
            e_done[l].record(stream)
            with torch.cuda.stream(s_out):
                s_out.wait_event(e_done[l])
                h_o[b].copy_(obuf[b][0], non_blocking=True)
                e_out[l] = ev()
                e_out[l].record(s_out)
        stream.wait_event(e_blk)                       # the suffix's queries (and L = 1)
        for l in range(L):
            nexus.suffix_attention(wl.cache, wl.d_pt, 2, wl.max_pages, [wl.T], [wl.R_split],
                                   wl.q_suf[l:l + 1], wl.o_suf[l:l + 1], wl.lse_suf[l:l + 1], HQ,
                                   l, l + 1, rows=[1], split_kv=0, workspace=wl.ws,
                                   workspace_bytes=wl.ws_bytes, stream=stream)
        e_suf = ev()
        e_suf.record(stream)
        with torch.cuda.stream(s_out):
            s_out.wait_event(e_suf)
            h_os.copy_(wl.o_suf, non_blocking=True)
        stream.wait_stream(s_out)
        stream.wait_stream(s_in)

    for _ in range(max(1, min(args.warmup, 2))):
        one()
    barrier()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        one()
    barrier()
    secs = max_over_ranks(time.perf_counter() - t0, dist, dev)
    per = secs / args.steps
    flops = wl.flops_pre + wl.flops_suf
    return {"value": job_throughput(flops, world, per * 1e3), "unit": "TFLOP/s",
            "ms_per_step": per * 1e3, "h2d_bytes_per_step": int(h2d),
            "d2h_bytes_per_step": int(d2h),
            "staging_huge_page_fraction": _huge_page_fraction([h_qall, h_oall, h_bk])}


if __name__ == "__main__":
    main()
