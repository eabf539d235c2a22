"""Benchmark of the DAR attention hot path on GB300.

One step = one decode step of the 160M-like workload (B32 H12 d64, context 4096,
w128, d_down 16, bf16): ``dar_cache_append`` of one token per sequence (the
token leaving the window is down-projected into its page) followed by
``dar_attn_decode``.  ``value`` is algorithmic bytes per step / device time
(GB/s, whole job).  The caches rotate over enough copies that the bytes
touched between two uses of one copy exceed 4x L2, so no step reads a warm L2.

Also reported on the same line: the decode kernel's roofline (live CUDA-event
duration of that kernel inside the timed region), an end-to-end number through
the public API with host buffers, the CPU oracle on a bounded sample, the SM
clocks seen during the timed region, and the 410M-like prefill (B8 H16 N8192
w512 d_down 16, bf16) in TFLOP/s.

``--impl reference`` times the CPU oracle (the reference arm of this build) on
the same workload and prints the same kind of line.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "decode GB/s & prefill TFLOP/s of DAR attention, % of GB300 roofline (1 GPU)"
# kernels of one timed step: the cache append, then the decode's prep and stream kernels
LAUNCHES_PER_STEP = 3
# DRAM bytes (read + write) of one decode_kernel<bf16,16,1> launch on the
# decode-160M workload, from an ncu capture of `python bench.py --only decode`
# (dram__bytes_read.sum + dram__bytes_write.sum); None whenever that kernel
# has changed since the capture.
DECODE_TRAFFIC_BYTES = 112_347_648 + 2_752_512
# multi-function-unit ex2 throughput per SM and the maximum SM clock (the
# prefill's exponential roofline)
MUFU_EX2_PER_CLK = 16
SM_MAX_MHZ = 2070.0


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), float(p["bf16_tflops"]), float(p.get("bf16_tflops_sustained", p["bf16_tflops"])), \
            "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


# ----------------------------------------------------------------------------- distributed

def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def init_dist(world, backend):
    import torch.distributed as dist
    if world > 1 and not dist.is_initialized():
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group(backend)
    return dist


def max_over_ranks(x: float, world: int, device=None) -> float:
    """Largest value of x over all ranks (the job's time is its slowest rank's)."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


# ----------------------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi clock / throttle samples while the timed region runs."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        self.out = ""
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.out, _ = self.proc.communicate()

    def summary(self):
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in (getattr(self, "out", "") or "").strip().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                smax.append(float(parts[1]))
            except ValueError:
                continue
            for name, val in zip(names, parts[4:8]):
                if val.lower() == "active":
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm)}


# ----------------------------------------------------------------------------- oracle (CPU) timing

def oracle_decode_sample(cfg, budget_s=12.0, nthreads=None):
    """Time the CPU oracle on whole sequences of the decode workload until about
    ``budget_s`` seconds are spent; returns (GB/s over the cache bytes of the
    sample, cores, description)."""
    import oracle
    from paper_2606_18587_gb300 import inputs as I
    from paper_2606_18587_gb300 import workloads as W
    nthreads = nthreads or os.cpu_count() or 1
    lens = I.decode_lengths(cfg)
    Dk, Uk, Dv, Uv = I.projections(cfg.seed, cfg.Hkv, cfg.d, cfg.dd)
    q = I.decode_query(cfg)
    spent, nbytes, nseq = 0.0, 0, 0
    for b in range(cfg.B):
        kb, vb = I.decode_history(cfg, b, int(lens[b]))
        t0 = time.perf_counter()
        oracle.decode(np.ascontiguousarray(q[b:b + 1]), kb[None], vb[None], lens[b:b + 1], Dk, Uk, Dv, Uv, cfg.w,
                      cfg.dtype, nthreads=nthreads)
        spent += time.perf_counter() - t0
        sub = I.Decode(cfg.name, cfg.seed, 1, cfg.Hq, cfg.Hkv, cfg.d, cfg.dd, cfg.w, cfg.dtype, L=int(lens[b]))
        nbytes += W.decode_step_bytes(sub, lens[b:b + 1])
        nseq += 1
        if spent >= budget_s:
            break
    return nbytes / spent / 1e9, nthreads, f"{nseq} of {cfg.B} sequences (all {cfg.Hq} heads), one decode step each"


def graph_kernel_times(torch, dar, wls, knew, vnew, outs, R, K, stream):
    """Per-call device time of dar_attn_decode and of dar_cache_append, each from
    a CUDA graph of K calls of that entry point alone (events between the
    kernels of the timed step would serialise them and add their own latency)."""
    res = []
    for which in ("decode", "append"):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for j in range(K):
                c = j % R
                wl = wls[c]
                if which == "decode":
                    dar.dar_attn_decode(wl.cache, wl.q, wl.Uk, wl.Uv, wl.workspace, out=outs[c])
                else:
                    dar.dar_cache_append(wl.cache, knew[c], vnew[c], wl.Dk, wl.Dv)
        g.replay()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        g.replay()
        b.record(stream)
        torch.cuda.synchronize()
        res.append([a.elapsed_time(b) / K] * K)
    return res[0], res[1]


# ----------------------------------------------------------------------------- GPU arm

def prefill_section(args, torch, W, I, dev, stream, tc_peak, peak_src):
    """Time the 410M-like prefill (B = --prefill-batch, 8 by default) and
    return its JSON object."""
    K, Wm = args.steps, args.warmup
    pcfg = I.PREFILL_410M
    if args.prefill_batch != pcfg.B:
        pcfg = I.Prefill(f"{pcfg.name} (B={args.prefill_batch})", pcfg.seed, args.prefill_batch, pcfg.Hq, pcfg.Hkv,
                         pcfg.N, pcfg.d, pcfg.dd, pcfg.w, pcfg.dtype)
    pw = W.PrefillWorkload(pcfg)
    flops = W.prefill_flops(pcfg)
    for _ in range(max(3, Wm)):
        pw.run()
    torch.cuda.synchronize()
    pk = max(3, min(K, 10))
    pev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(pk)]
    for a, b in pev:
        a.record(stream)
        pw.run()
        b.record(stream)
    torch.cuda.synchronize()
    p_ms = float(np.mean([a.elapsed_time(b) for a, b in pev]))
    p_tflops = flops / (p_ms * 1e-3) / 1e12
    # The prefill is bound by the exponentials of the softmax (one per causal
    # (query, key) pair), not by its small contractions: 16 ex2 per clock per
    # SM on the multi-function units, at the maximum SM clock.
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    exps = W.prefill_exps(pcfg)
    exp_rate = exps / (p_ms * 1e-3) / 1e9
    exp_peak = sms * MUFU_EX2_PER_CLK * SM_MAX_MHZ * 1e6 / 1e9
    prefill = {"workload": pcfg.name, "tflops": round(p_tflops, 2), "ms": round(p_ms, 4),
               "flops_per_call": flops, "exps_per_call": exps,
               "roofline": {"bound": "alu", "achieved": round(exp_rate, 1), "peak": round(exp_peak, 1),
                            "unit": "Gexp/s", "frac": round(exp_rate / exp_peak, 4), "traffic": None,
                            "peak_source": f"{sms} SMs x {MUFU_EX2_PER_CLK} ex2/clk x {SM_MAX_MHZ:.0f} MHz (nominal)"},
               "tensor": {"achieved": round(p_tflops, 2), "peak": tc_peak, "unit": "TFLOP/s",
                          "frac": round(p_tflops / tc_peak, 4), "peak_source": f"{peak_src} bf16 dense (burst)"}}

    return prefill



def run_ours(args, world, rank, local):
    import torch
    from paper_2606_18587_gb300 import dar
    from paper_2606_18587_gb300 import inputs as I
    from paper_2606_18587_gb300 import workloads as W

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    init_dist(world, "nccl")
    hbm_peak, tc_peak, tc_sus, peak_src = load_peaks()
    if args.only == "prefill":  # profiling aid: the prefill alone
        pre = prefill_section(args, torch, W, I, dev, torch.cuda.current_stream(), tc_peak, peak_src)
        if rank == 0:
            print(json.dumps({"metric": "prefill (profiling run)", "prefill": pre}), flush=True)
        return
    cfg = I.DECODE_160M
    K, Wm = args.steps, args.warmup

    # rotating caches: each step uses the next copy, so between two uses of one copy
    # the other copies (more than 4x L2 in total) pass through the memory system
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    one = W.decode_step_bytes(cfg, I.decode_lengths(cfg))
    R = max(2, int(np.ceil(4 * l2 / one)) + 1)
    wls = [W.DecodeWorkload(cfg, extra_tokens=2 * K + Wm + 8) for _ in range(R)]
    knew, vnew = [], []
    for s in range(R):
        kh, vh = I.decode_new_tokens(cfg, s)
        knew.append(W.upload(kh, cfg.dtype))
        vnew.append(W.upload(vh, cfg.dtype))
    outs = [torch.empty_like(wl.q) for wl in wls]
    stream = torch.cuda.current_stream()

    def step(i):
        wl = wls[i % R]
        dar.dar_decode_step(wl.cache, knew[i % R], vnew[i % R], wl.Dk, wl.Dv, wl.q, wl.Uk, wl.Uv, wl.workspace,
                            out=outs[i % R])

    for i in range(Wm):
        step(i)
    torch.cuda.synchronize()

    # The timed region is one CUDA graph of K steps, so the device runs them back
    # to back with no host launch latency between kernels (and the kernels of
    # one step overlap as their programmatic launches allow).
    # every replay first restores the lengths, so each replay appends at the same
    # positions and reads the same bytes (the restore copies are inside the timed region)
    lens0 = [wl.cache.seq_lens.clone() for wl in wls]
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        cap = torch.cuda.current_stream()
        for c in range(R):
            wls[c].cache.seq_lens.copy_(lens0[c], non_blocking=True)
        for j in range(K):
            c = j % R
            wl = wls[c]
            dar.dar_decode_step(wl.cache, knew[c], vnew[c], wl.Dk, wl.Dv, wl.q, wl.Uk, wl.Uv, wl.workspace,
                                out=outs[c])
    # warm the graph and size the soak
    graph.replay()
    torch.cuda.synchronize()
    w0, w1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    w0.record(stream)
    for _ in range(3):
        graph.replay()
    w1.record(stream)
    torch.cuda.synchronize()
    soak = max(1, int(args.soak_seconds / (w0.elapsed_time(w1) / 3 * 1e-3)))
    lens_at = [x.cpu().numpy().astype(np.int64) for x in lens0]

    # algorithmic bytes of the K steps of one replay
    step_bytes, dec_bytes = [], []
    for j in range(K):
        c = j % R
        L_before = lens_at[c] + j // R
        step_bytes.append(W.append_step_bytes(cfg, L_before) + W.decode_step_bytes(cfg, L_before + 1))
        dec_bytes.append(W.decode_step_bytes(cfg, L_before + 1))

    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier(world)
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        # untimed soak of the same graph so the sampled clocks reflect this load,
        # then exactly K timed steps (one replay)
        for _ in range(soak):
            graph.replay()
        torch.cuda.synchronize()
        barrier(world)
        start.record(stream)
        graph.replay()
        stop.record(stream)
        torch.cuda.synchronize()
        barrier(world)
    total_ms = max_over_ranks(start.elapsed_time(stop), world, dev)
    steps_done = K
    # per-call durations of the two entry points, each from a graph of its own
    dec_ms, app_ms = graph_kernel_times(torch, dar, wls, knew, vnew, outs, R, K, stream)
    status = sum(wl.cache.device_status() for wl in wls)
    if status:
        raise RuntimeError(f"device status {status} during the benchmark")

    value = world * sum(step_bytes) / (total_ms * 1e-3) / 1e9
    dec_gbs = float(np.mean(dec_bytes)) / (float(np.mean(dec_ms)) * 1e-3) / 1e9

    # ---- end to end through the public API: host buffers, copies inside the timed region.
    # A step's inputs (k_new, v_new, q) sit in one pinned host buffer and go to
    # the device in one copy; the API is called on views of the device copy.
    nk, nv, nq = knew[0].numel(), vnew[0].numel(), wls[0].q.numel()
    h_in, d_in = [], []
    for c in range(R):
        h = torch.cat([knew[c].reshape(-1), vnew[c].reshape(-1), wls[c].q.reshape(-1)]).cpu().pin_memory()
        h_in.append(h)
        d_in.append(torch.empty_like(h, device=dev))
    views = [(d[:nk].view(knew[0].shape), d[nk:nk + nv].view(vnew[0].shape), d[nk + nv:].view(wls[0].q.shape))
             for d in d_in]
    hout = [torch.empty(o.shape, dtype=o.dtype, pin_memory=True) for o in outs]
    lens_e2e = [W.download(wl.cache.seq_lens).astype(np.int64) for wl in wls]
    e2e_bytes = []
    for j in range(K):
        L_before = lens_e2e[j % R] + j // R
        e2e_bytes.append(W.append_step_bytes(cfg, L_before) + W.decode_step_bytes(cfg, L_before + 1))
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier(world)
    torch.cuda.synchronize()
    e0.record(stream)
    for j in range(K):
        c = j % R
        wl = wls[c]
        d_in[c].copy_(h_in[c], non_blocking=True)
        k_c, v_c, q_c = views[c]
        dar.dar_decode_step(wl.cache, k_c, v_c, wl.Dk, wl.Dv, q_c, wl.Uk, wl.Uv, wl.workspace, out=outs[c])
        hout[c].copy_(outs[c], non_blocking=True)
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1), world, dev)
    e2e_val = world * sum(e2e_bytes) / (e2e_ms * 1e-3) / 1e9
    h2d = h_in[0].numel() * h_in[0].element_size()
    d2h = outs[0].numel() * outs[0].element_size()

    prefill = None if args.only == "decode" else prefill_section(args, torch, W, I, dev, stream, tc_peak, peak_src)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        gbs, cores, sample = oracle_decode_sample(cfg, budget_s=args.cpu_budget)
        cpu = {"value": round(gbs, 4), "unit": "GB/s", "cores": cores, "kind": "oracle", "sample": sample}

    if rank == 0:
        line = {
            "metric": METRIC, "value": round(value, 2), "unit": "GB/s", "n_gpus": world, "steps": steps_done, "warmup": Wm,
            "ms_per_step": round(total_ms / steps_done, 5), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic (seeded N(0,1) keys/values/queries)",
            "config": {"workload": cfg.name, "B": cfg.B, "Hq": cfg.Hq, "Hkv": cfg.Hkv, "context": cfg.L,
                       "w": cfg.w, "d": cfg.d, "d_down": cfg.dd, "step": "append 1 token + decode",
                       "l2": f"{R} rotating cache copies ({R * one / 1e6:.0f} MB > 4x L2 {l2 / 1e6:.0f} MB)",
                       "parallelism": f"{world} independent replicas" if world > 1 else "single GPU"},
            "clocks": clk.summary(),
            "e2e": {"value": round(e2e_val, 2), "unit": "GB/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
            "gpu_launches": LAUNCHES_PER_STEP * steps_done,
            "roofline": {"bound": "hbm", "achieved": round(dec_gbs, 1), "peak": hbm_peak, "unit": "GB/s",
                         "frac": round(dec_gbs / hbm_peak, 4), "traffic": DECODE_TRAFFIC_BYTES,
                         "kernel": "dar_attn_decode (decode_prep_kernel + decode_kernel<bf16,16,1>)",
                         "bytes_per_launch": int(np.mean(dec_bytes)),
                         "us_per_launch": round(1e3 * float(np.mean(dec_ms)), 3),
                         "peak_source": f"{peak_src} HBM copy"},
            "append_us_per_launch": round(1e3 * float(np.mean(app_ms)), 3),
            "prefill": prefill,
        }
        if cpu:
            line["cpu_baseline"] = cpu
        print(json.dumps(line), flush=True)


# ----------------------------------------------------------------------------- reference arm

def run_reference(args, world, rank, local):
    """The CPU oracle on the same decode workload: each step is one whole
    sequence's decode step (all heads), on all host cores."""
    if world > 1:
        init_dist(world, "gloo")
        if rank != 0:
            barrier(world)
            return
    from paper_2606_18587_gb300 import inputs as I
    cfg = I.DECODE_160M
    budget = max(1.0, args.cpu_budget / max(1, args.steps + args.warmup))
    for _ in range(args.warmup):
        oracle_decode_sample(cfg, budget_s=0.0)
    vals = []
    t0 = time.perf_counter()
    for _ in range(args.steps):
        gbs, cores, sample = oracle_decode_sample(cfg, budget_s=budget)
        vals.append(gbs)
    wall = time.perf_counter() - t0
    v = float(np.mean(vals))
    line = {"impl": "reference", "metric": METRIC, "value": round(v, 4), "unit": "GB/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(1e3 * wall / args.steps, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded N(0,1) keys/values/queries)",
            "config": {"workload": cfg.name, "B": cfg.B, "Hq": cfg.Hq, "Hkv": cfg.Hkv, "context": cfg.L,
                       "w": cfg.w, "d": cfg.d, "d_down": cfg.dd, "step": "one decode step of a sample"},
            "cpu_baseline": {"value": round(v, 4), "unit": "GB/s", "cores": os.cpu_count(), "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": round(v, 4), "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    if world > 1:
        barrier(world)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--cpu-budget", type=float, default=12.0, help="seconds of oracle time for the CPU baseline")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--only", choices=["all", "decode", "prefill"], default="all",
                    help="profiling aid: run only the decode step or only the prefill")
    ap.add_argument("--prefill-batch", type=int, default=8, help="batch of the prefill workload")
    ap.add_argument("--soak-seconds", type=float, default=1.0,
                    help="untimed replays of the step graph just before the timed region (clock sampling)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    world, rank, local = dist_env()
    if args.impl == "reference":
        run_reference(args, world, rank, local)
    else:
        run_ours(args, world, rank, local)


if __name__ == "__main__":
    main()
