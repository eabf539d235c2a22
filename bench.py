"""Benchmark of the DAR attention hot path on GB300.

One step = one serving step of the 160M-like decode workload (B32 H12 d64,
context 4096, w128, d_down 16, bf16): ``dar_decode_step`` appends one token to
every sequence (the token leaving the window is down-projected into its page)
and decodes.  ``value`` is the algorithmic bytes of K steps / the device time
of one CUDA-graph replay of those K steps (GB/s, whole job).  The caches rotate
over enough copies that the bytes touched between two uses of one copy exceed
4x L2; before the timed replay the caches are restored to their starting state
(outside the timed region) and L2 is flushed.  After it, the outputs of the
timed steps are checked against the CPU oracle and against an eager call.

Also reported on the same line: the decode kernel's roofline (CUDA-event time
of graphs of decode calls alone), an end-to-end number through the public API
from pinned host buffers (the step's inputs copied in and its output copied
out every step, copies overlapped with the previous step's kernels), the
410M-like prefill (B8 H16 N8192 w512 d_down 16) against its exponential and
tensor-core rooflines, GB/s of the ragged GQA 1B-like decode and of the 16
points of the window x d_down sweep, the CPU oracle on bounded samples (all
host cores, and one thread), and the SM clocks seen while each part ran.

``--impl reference`` times the CPU oracle (the reference arm of this build) on
the same workload and prints the same kind of line.
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

METRIC = "decode GB/s & prefill TFLOP/s of DAR attention, % of GB300 roofline (1 GPU)"
# kernels of one timed step: the cache append, then the decode's prep and stream kernels
LAUNCHES_PER_STEP = 3
# DRAM bytes (read + write) of one decode_kernel<bf16,16,1> launch on the
# decode-160M workload, from an ncu capture of `python bench.py --only decode`
# (dram__bytes_read.sum + dram__bytes_write.sum); None whenever that kernel
# has changed since the capture.
DECODE_TRAFFIC_BYTES = 112_347_648 + 2_752_512
# ex2 results per clock per SM on the multi-function unit, measured on GB300
# with a throughput probe (f32 and packed bf16x2 alike), and the maximum SM
# clock: the prefill's exponential roofline
MUFU_EX2_PER_CLK = 32
SM_MAX_MHZ = 2070.0
NOMINAL_HBM_GBS = 8000.0
TOL_BF16 = 2e-2


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
    """nvidia-smi clock / throttle samples while a timed region runs."""

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


def oracle_prefill_sample(cfg, budget_s=5.0, nthreads=None):
    """Time the CPU oracle on rows of one head of a prefill workload (positions
    spread over the sequence) until about ``budget_s`` seconds are spent;
    returns (TFLOP/s of the rows' algorithmic work, cores, description)."""
    import oracle
    from paper_2606_18587_gb300 import inputs as I
    nthreads = nthreads or os.cpu_count() or 1
    s = cfg.seed
    q = I.normal_array(s, I.S_Q, (1, 1, cfg.N, cfg.d), dtype=cfg.dtype)
    k = I.normal_array(s, I.S_K, (1, 1, cfg.N, cfg.d), dtype=cfg.dtype)
    v = I.normal_array(s, I.S_V, (1, 1, cfg.N, cfg.d), dtype=cfg.dtype)
    Dk, Uk, Dv, Uv = (x[:1] for x in I.projections(s, cfg.Hkv, cfg.d, cfg.dd))
    rng = np.random.default_rng(0)
    spent, flops, nrows = 0.0, 0.0, 0
    while spent < budget_s and nrows < 4096:
        pos = np.sort(rng.integers(0, cfg.N, 16))
        rows = np.array([(0, 0, int(i)) for i in pos])
        t0 = time.perf_counter()
        oracle.prefill(q, k, v, Dk, Uk, Dv, Uv, cfg.w, cfg.dtype, rows=rows, nthreads=nthreads)
        spent += time.perf_counter() - t0
        for i in pos:
            loc = min(int(i) + 1, cfg.w)
            flops += 4 * cfg.d * loc + 4 * cfg.dd * (int(i) + 1 - loc) + 4 * cfg.d * cfg.dd
        nrows += len(pos)
    return flops / spent / 1e12, nthreads, f"{nrows} rows of head (0, 0) at random positions (whole rows, Eq. 1-4)"


# ----------------------------------------------------------------------------- GPU helpers

def flush_l2(torch, dev, nbytes):
    """Write a buffer larger than L2 so no earlier data stays cached."""
    buf = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    buf.fill_(1)
    del buf


def clone_cache(dar, cache):
    """A device copy of a cache (same shape, same page table, same contents)."""
    c = dar.DarCache(cache.B, cache.Hkv, cache.d_down, cache.w, cache.max_pages_per_seq, cache.num_pages,
                     dtype=cache.dtype, block_table=cache.block_table, device=cache.win_k.device)
    for name in ("win_k", "win_v", "pool_kd", "pool_vd", "seq_lens"):
        getattr(c, name).copy_(getattr(cache, name))
    return c


def graph_of(torch, fn, K):
    """Capture K calls fn(j) in one CUDA graph."""
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for j in range(K):
            fn(j)
    return g


def time_graph(torch, g, stream, before=None):
    """Device time (ms) of one replay, after one untimed replay."""
    if before:
        before()
    g.replay()
    torch.cuda.synchronize()
    if before:
        before()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    a.record(stream)
    g.replay()
    b.record(stream)
    torch.cuda.synchronize()
    return a.elapsed_time(b)


def decode_only_point(torch, dar, I, W, cfg, K, l2, dev, stream, hbm_peak, direct=False):
    """GB/s of graph-timed dar_attn_decode calls on one decode workload (the
    cache is read, never written, so replays are identical); caches rotate
    over enough copies to exceed 4x L2.  direct: dar_attn_decode_direct (the
    global path of Sec. 5's direct variant; same cache bytes)."""
    wl = W.DecodeWorkload(cfg)
    lens = W.download(wl.cache.seq_lens).astype(np.int64)
    nbytes = W.decode_step_bytes(cfg, lens)
    R = 1 if nbytes > 4 * l2 else int(math.ceil(4 * l2 / nbytes)) + 1
    caches = [wl.cache] + [clone_cache(dar, wl.cache) for _ in range(R - 1)]
    outs = [torch.empty_like(wl.q) for _ in range(R)]
    ws = [wl.workspace] + [dar.decode_workspace(c, cfg.Hq) for c in caches[1:]]
    if direct:
        qd = W.upload(I.direct_queries(cfg), cfg.dtype)
        g = graph_of(torch, lambda j: dar.dar_attn_decode_direct(caches[j % R], wl.q, qd, wl.Uv, ws[j % R],
                                                                 out=outs[j % R]), K)
    else:
        g = graph_of(torch, lambda j: dar.dar_attn_decode(caches[j % R], wl.q, wl.Uk, wl.Uv, ws[j % R],
                                                          out=outs[j % R]), K)
    ms = time_graph(torch, g, stream, before=lambda: flush_l2(torch, dev, 2 * l2))
    us = 1e3 * ms / K
    gbs = nbytes / (us * 1e-6) / 1e9
    status = sum(c.device_status() for c in caches)
    res = {"workload": cfg.name, "bytes_per_call": int(nbytes), "us_per_call": round(us, 3), "gbs": round(gbs, 1),
           "frac_measured": round(gbs / hbm_peak, 4), "frac_nominal": round(gbs / NOMINAL_HBM_GBS, 4),
           "copies": R}
    del g, caches, outs, ws, wl
    torch.cuda.empty_cache()
    if status:
        raise RuntimeError(f"device status {status} on {cfg.name}")
    return res


# ----------------------------------------------------------------------------- GPU arm: sections

def prefill_section(args, torch, dar, W, I, dev, stream, tc_peak, peak_src, local):
    """Time the 410M-like prefill (B = --prefill-batch, 8 by default), check
    sampled rows against the oracle, and return its JSON object."""
    import oracle
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
    with ClockSampler(local) as clk:
        t_end = time.perf_counter() + args.soak_seconds  # untimed calls first, so the clocks see this load
        while time.perf_counter() < t_end:
            pw.run()
            torch.cuda.synchronize()
        pev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(pk)]
        for a, b in pev:
            a.record(stream)
            pw.run()
            b.record(stream)
        torch.cuda.synchronize()
    times = [a.elapsed_time(b) for a, b in pev]
    p_ms = float(np.median(times))
    # the Eq. 1 pre-pass alone (keys and values), for the split of the call
    kd = torch.empty((pcfg.B, pcfg.Hkv, pcfg.N, pcfg.dd), dtype=pw.q.dtype, device=dev)
    dp_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(pk)]
    for a, b in dp_ev:
        a.record(stream)
        dar.dar_down_project(pw.k, pw.Dk, out=kd)
        dar.dar_down_project(pw.v, pw.Dv, out=kd)
        b.record(stream)
    torch.cuda.synchronize()
    dp_ms = float(np.median([a.elapsed_time(b) for a, b in dp_ev]))
    # sampled rows of the last timed call against the oracle
    rng = np.random.default_rng(1)
    x = pw.host
    rows = np.array([(int(rng.integers(pcfg.B)), int(rng.integers(pcfg.Hq)), int(i))
                     for i in [0, pcfg.w - 1, pcfg.w, pcfg.N - 1] + list(rng.integers(0, pcfg.N, 4))])
    want = oracle.prefill(x["q"], x["k"], x["v"], x["Dk"], x["Uk"], x["Dv"], x["Uv"], pcfg.w, pcfg.dtype, rows=rows)
    got = W.to_f64(W.download(pw.out), pcfg.dtype)[rows[:, 0], rows[:, 1], rows[:, 2]]
    err = float(np.abs(got - want).max())
    if not err <= TOL_BF16:
        raise RuntimeError(f"prefill output differs from the oracle: max-abs {err}")
    p_tflops = flops / (p_ms * 1e-3) / 1e12
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    exps = W.prefill_exps(pcfg)
    exp_rate = exps / (p_ms * 1e-3) / 1e9
    exp_peak = sms * MUFU_EX2_PER_CLK * SM_MAX_MHZ * 1e6 / 1e9
    attn_ms = max(p_ms - dp_ms, 1e-6)
    return {"workload": pcfg.name, "ms": round(p_ms, 4), "tflops": round(p_tflops, 2),
            "flops_per_call": flops, "exps_per_call": exps, "oracle_max_abs_err": round(err, 5),
            "down_project_ms": round(dp_ms, 4), "attention_ms_est": round(attn_ms, 4),
            "roofline": {"bound": "alu", "achieved": round(exp_rate, 1), "peak": round(exp_peak, 1),
                         "unit": "Gexp/s", "frac": round(exp_rate / exp_peak, 4), "traffic": None,
                         "attention_frac_est": round(exps / (attn_ms * 1e-3) / 1e9 / exp_peak, 4),
                         "peak_source": f"{sms} SMs x {MUFU_EX2_PER_CLK} ex2/clk (measured probe) x {SM_MAX_MHZ:.0f} MHz"},
            "tensor": {"achieved": round(p_tflops, 2), "peak": tc_peak, "unit": "TFLOP/s",
                       "frac": round(p_tflops / tc_peak, 4), "peak_source": f"{peak_src} bf16 dense (burst)"},
            "clocks": clk.summary()}


def latent_point(torch, dar, I, W, cfg, K, l2, dev, stream, hbm_peak):
    """GB/s of graph-timed dar_latent_decode calls on a latent-form workload
    (one bottleneck per token shared by every head); cache copies rotate so
    the bytes between two uses of one copy exceed 4x L2.  The first call's
    output is checked against the oracle on two sequences."""
    import oracle
    wl = W.LatentDecodeWorkload(cfg, keep_history=True)
    nbytes = W.latent_decode_bytes(cfg, wl.lens)
    R = 1 if nbytes > 4 * l2 else int(math.ceil(4 * l2 / nbytes)) + 1
    caches = [wl.cache]
    for _ in range(R - 1):
        c = dar.DarLatentCache(cfg.B, cfg.Hkv, cfg.D, cfg.dl, cfg.w, wl.cache.max_pages_per_seq,
                               wl.cache.num_pages, block_table=wl.cache.block_table, device=dev)
        for name in ("win_k", "win_v", "pool_c", "seq_lens"):
            getattr(c, name).copy_(getattr(wl.cache, name))
        caches.append(c)
    outs = [torch.empty_like(wl.q) for _ in range(R)]
    ws = [wl.workspace] + [dar.latent_decode_workspace(c, cfg.Hq) for c in caches[1:]]
    g = graph_of(torch, lambda j: dar.dar_latent_decode(caches[j % R], wl.q, wl.A_K, wl.A_V, ws[j % R],
                                                        out=outs[j % R]), K)
    ms = time_graph(torch, g, stream, before=lambda: flush_l2(torch, dev, 2 * l2))
    us = 1e3 * ms / K
    gbs = nbytes / (us * 1e-6) / 1e9
    status = sum(c.device_status() for c in caches)
    seqs = [0, cfg.B - 1]
    k, v, h = wl.history_arrays(seqs)
    Wdown, Wup, WK, WV = wl.proj_host
    heads = [(i, hq) for i in range(2) for hq in range(cfg.Hq)]
    want = oracle.latent_decode(np.ascontiguousarray(wl.q_host[seqs]), k, v, h, wl.lens[seqs], Wdown, Wup, WK, WV,
                                cfg.w, "bf16", heads=heads)
    got = W.to_f64(W.download(outs[0]), "bf16")[seqs]
    err = float(np.abs(got - want).max())
    res = {"workload": cfg.name, "bytes_per_call": int(nbytes), "us_per_call": round(us, 3), "gbs": round(gbs, 1),
           "frac_measured": round(gbs / hbm_peak, 4), "frac_nominal": round(gbs / NOMINAL_HBM_GBS, 4),
           "copies": R, "oracle_max_abs_err": round(err, 5)}
    del g, caches, outs, ws, wl
    torch.cuda.empty_cache()
    if status:
        raise RuntimeError(f"device status {status} on {cfg.name}")
    if not err <= TOL_BF16:
        raise RuntimeError(f"latent decode output differs from the oracle: max-abs {err}")
    return res


def direct_prefill_point(args, torch, dar, W, I, dev, stream):
    """The 410M-like prefill with the direct global path of Sec. 5
    (dar_attn_prefill_direct): median CUDA-event time of K calls, sampled rows
    checked against the oracle."""
    import oracle
    pcfg = I.PREFILL_410M
    pw = W.PrefillWorkload(pcfg)
    qd_host = I.direct_queries(pcfg)
    qd = W.upload(qd_host, pcfg.dtype)

    def call():
        dar.dar_attn_prefill_direct(pw.q, qd, pw.k, pw.v, pw.Dk, pw.Dv, pw.Uv, pcfg.w, out=pw.out,
                                    workspace=pw.workspace, stream=stream)

    for _ in range(3):
        call()
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(max(3, min(args.steps, 10)))]
    for a, b in ev:
        a.record(stream)
        call()
        b.record(stream)
    torch.cuda.synchronize()
    ms = float(np.median([a.elapsed_time(b) for a, b in ev]))
    rng = np.random.default_rng(2)
    rows = np.array([(int(rng.integers(pcfg.B)), int(rng.integers(pcfg.Hq)), int(i))
                     for i in [0, pcfg.w - 1, pcfg.w, pcfg.N - 1] + list(rng.integers(0, pcfg.N, 4))])
    x = pw.host
    want = oracle.prefill_direct(x["q"], qd_host, x["k"], x["v"], x["Dk"], x["Dv"], x["Uv"], pcfg.w, pcfg.dtype,
                                 rows=rows)
    got = W.to_f64(W.download(pw.out), pcfg.dtype)[rows[:, 0], rows[:, 1], rows[:, 2]]
    err = float(np.abs(got - want).max())
    if not err <= TOL_BF16:
        raise RuntimeError(f"direct prefill output differs from the oracle: max-abs {err}")
    flops = W.prefill_flops(pcfg)  # the direct path does the same contractions, minus the q Uk^T lift
    return {"workload": pcfg.name, "ms": round(ms, 4), "tflops": round(flops / (ms * 1e-3) / 1e12, 2),
            "exps_per_call": W.prefill_exps(pcfg), "oracle_max_abs_err": round(err, 5)}


def backward_point(args, torch, dar, W, I, dev, stream, tc_peak=None):
    """The backward pass (Sec. 2.3 training) of the 410M-like prefill:
    dar_attn_backward after one forward, median CUDA-event time of a few calls.
    The bf16 contractions run on the tensor cores: the roofline is the bf16
    dense peak, with the exponential bound (two per causal pair: P is
    recomputed by the dq and the dk/dv kernels) beside it.  The gradients must
    be finite and bit-identical across calls; their values are checked against
    the oracle in the GPU tests."""
    pcfg = I.PREFILL_410M
    pw = W.PrefillWorkload(pcfg)
    pw.run()
    dout = W.upload(I.normal_array(pcfg.seed, I.S_QD, (pcfg.B, pcfg.Hq, pcfg.N, pcfg.d), dtype=pcfg.dtype, sub=1),
                    pcfg.dtype)
    ws = torch.empty(dar.dar_attn_backward_workspace_bytes(pw.q.dtype, pcfg.B, pcfg.Hq, pcfg.Hkv, pcfg.N, pcfg.dd),
                     dtype=torch.uint8, device=dev)
    grads = dar.dar_attn_backward(pw.q, pw.k, pw.v, pw.Dk, pw.Uk, pw.Dv, pw.Uv, pw.out, dout, pcfg.w, workspace=ws,
                                  stream=stream)
    first = {n: t.clone() for n, t in grads.items()}
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(3)]
    for a, b in ev:
        a.record(stream)
        dar.dar_attn_backward(pw.q, pw.k, pw.v, pw.Dk, pw.Uk, pw.Dv, pw.Uv, pw.out, dout, pcfg.w, workspace=ws,
                              grads=grads, stream=stream)
        b.record(stream)
    torch.cuda.synchronize()
    ms = float(np.median([a.elapsed_time(b) for a, b in ev]))
    for n, t in grads.items():
        if not bool(torch.isfinite(t.float()).all()) or not torch.equal(t, first[n]):
            raise RuntimeError(f"backward gradient {n} is not finite or not repeatable")
    flops = W.prefill_backward_flops(pcfg)
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    peak = tc_peak if tc_peak else load_peaks()[1]
    tf = flops / (ms * 1e-3) / 1e12
    exps = 2 * W.prefill_exps(pcfg)
    exp_ms = exps / (sms * MUFU_EX2_PER_CLK * SM_MAX_MHZ * 1e6) * 1e3
    return {"workload": pcfg.name, "ms": round(ms, 3), "tflops": round(tf, 2), "flops_per_call": flops,
            "roofline": {"bound": "tensor", "achieved": round(tf, 2), "peak": peak, "unit": "TFLOP/s",
                         "frac": round(tf / peak, 4), "peak_source": "measured bf16 dense (burst)",
                         "exp_bound_ms": round(exp_ms, 3), "tensor_bound_ms": round(flops / peak / 1e9, 3),
                         "frac_of_larger_bound": round(max(exp_ms, flops / peak / 1e9) / ms, 4)}}


def verify_steps(torch, dar, oracle, I, W, cfg, wls, outs, knew_host, vnew_host, n_appended, R):
    """The timed graph's outputs: for every rotating copy, the last step's
    output equals an eager decode of the same state bit for bit, and sequence
    0 (every head) matches the oracle on history + appended tokens."""
    worst = 0.0
    lens0 = I.decode_lengths(cfg)
    Dk, Uk, Dv, Uv = I.projections(cfg.seed, cfg.Hkv, cfg.d, cfg.dd)
    kb, vb = I.decode_history(cfg, 0, int(lens0[0]))
    for c in range(min(R, len(n_appended))):
        if n_appended[c][1] == 0:  # no step of the timed replay used this copy
            continue
        wl = wls[c]
        eager = dar.dar_attn_decode(wl.cache, wl.q, wl.Uk, wl.Uv, wl.workspace)
        torch.cuda.synchronize()
        if not np.array_equal(W.download(eager), W.download(outs[c])):
            raise RuntimeError(f"timed graph output of cache copy {c} differs from an eager decode of the same state")
        n = sum(n_appended[c])
        k = np.concatenate([kb] + [knew_host[c][0, :, :1]] * n, axis=1)[None]
        v = np.concatenate([vb] + [vnew_host[c][0, :, :1]] * n, axis=1)[None]
        want = oracle.decode(np.ascontiguousarray(wl.q_host[:1]), np.ascontiguousarray(k), np.ascontiguousarray(v),
                             np.array([lens0[0] + n]), Dk, Uk, Dv, Uv, cfg.w, cfg.dtype)
        got = W.to_f64(W.download(outs[c]), cfg.dtype)[:1]
        worst = max(worst, float(np.abs(got - want).max()))
    if not worst <= TOL_BF16:
        raise RuntimeError(f"timed graph output differs from the oracle: max-abs {worst}")
    return worst


def run_ours(args, world, rank, local):
    import torch
    import oracle
    from paper_2606_18587_gb300 import dar
    from paper_2606_18587_gb300 import inputs as I
    from paper_2606_18587_gb300 import workloads as W

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    init_dist(world, "nccl")
    hbm_peak, tc_peak, tc_sus, peak_src = load_peaks()
    stream = torch.cuda.current_stream()
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    if args.only == "latent":  # profiling aid: the latent-form decode alone
        res = [latent_point(torch, dar, I, W, c, args.steps, l2, dev, stream, hbm_peak)
               for c in (I.DECODE_160M_LATENT, I.DECODE_1B_LATENT)]
        if rank == 0:
            print(json.dumps({"metric": "latent decode (profiling run)", "latent_form": res}), flush=True)
        return
    if args.only == "prefill":  # profiling aid: the prefill alone
        pre = prefill_section(args, torch, dar, W, I, dev, stream, tc_peak, peak_src, local)
        if rank == 0:
            print(json.dumps({"metric": "prefill (profiling run)", "prefill": pre}), flush=True)
        return
    cfg = I.DECODE_160M
    K, Wm = args.steps, args.warmup

    # rotating caches: each step uses the next copy, so between two uses of one copy
    # the other copies (more than 4x L2 in total) pass through the memory system
    one = W.decode_step_bytes(cfg, I.decode_lengths(cfg))
    R = max(2, int(np.ceil(4 * l2 / one)) + 1)
    wls = [W.DecodeWorkload(cfg, extra_tokens=Wm + 6 * K + 16) for _ in range(R)]
    knew_host, vnew_host, knew, vnew = [], [], [], []
    for s in range(R):
        kh, vh = I.decode_new_tokens(cfg, s)
        knew_host.append(kh)
        vnew_host.append(vh)
        knew.append(W.upload(kh, cfg.dtype))
        vnew.append(W.upload(vh, cfg.dtype))
    outs = [torch.empty_like(wl.q) for wl in wls]

    def step(j):
        c = j % R
        wl = wls[c]
        dar.dar_decode_step(wl.cache, knew[c], vnew[c], wl.Dk, wl.Dv, wl.q, wl.Uk, wl.Uv, wl.workspace, out=outs[c])

    for i in range(Wm):
        step(i)
    torch.cuda.synchronize()

    # The timed region is one CUDA graph of K steps, so the device runs them back
    # to back with no host launch latency between kernels (the kernels of one
    # step overlap as their programmatic launches allow).  A second graph puts
    # every cache back to the state the steps start from (lengths and ring), so
    # each replay appends at the same positions and reads the same bytes; it
    # runs before the timed region, followed by an L2 flush.
    saved = [[t.clone() for t in (wl.cache.seq_lens, wl.cache.win_k, wl.cache.win_v)] for wl in wls]
    restore = torch.cuda.CUDAGraph()
    with torch.cuda.graph(restore):
        for wl, sv in zip(wls, saved):
            for dst, src in zip((wl.cache.seq_lens, wl.cache.win_k, wl.cache.win_v), sv):
                dst.copy_(src, non_blocking=True)
    steps_graph = graph_of(torch, step, K)

    def fresh():
        restore.replay()
        flush_l2(torch, dev, 2 * l2)

    fresh()
    steps_graph.replay()
    torch.cuda.synchronize()
    w0, w1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    w0.record(stream)
    steps_graph.replay()
    w1.record(stream)
    torch.cuda.synchronize()
    soak = max(1, int(args.soak_seconds / (w0.elapsed_time(w1) * 1e-3)))
    lens_at = [x[0].cpu().numpy().astype(np.int64) for x in saved]

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
        # then exactly K timed steps (one replay) from the restored state
        for _ in range(soak):
            restore.replay()
            steps_graph.replay()
        fresh()
        torch.cuda.synchronize()
        barrier(world)
        start.record(stream)
        steps_graph.replay()
        stop.record(stream)
        torch.cuda.synchronize()
        barrier(world)
    total_ms = max_over_ranks(start.elapsed_time(stop), world, dev)
    status = sum(wl.cache.device_status() for wl in wls)
    if status:
        raise RuntimeError(f"device status {status} during the benchmark")
    # tokens each copy has appended since it was filled: warm-up steps, then this replay's
    n_appended = [(len(range(c, Wm, R)), len(range(c, K, R))) for c in range(R)]
    verify_err = verify_steps(torch, dar, oracle, I, W, cfg, wls, outs, knew_host, vnew_host, n_appended, R)

    value = world * sum(step_bytes) / (total_ms * 1e-3) / 1e9

    # ---- per-call device times of the two parts, each from a graph of K calls
    # of that entry point alone (the decode reads but never writes the cache)
    dec_graph = graph_of(torch, lambda j: dar.dar_attn_decode(wls[j % R].cache, wls[j % R].q, wls[j % R].Uk,
                                                              wls[j % R].Uv, wls[j % R].workspace,
                                                              out=outs[j % R]), K)
    dec_ms = time_graph(torch, dec_graph, stream, before=lambda: flush_l2(torch, dev, 2 * l2)) / K
    dec_gbs = float(np.mean(dec_bytes)) / (dec_ms * 1e-3) / 1e9
    app_graph = graph_of(torch, lambda j: dar.dar_cache_append(wls[j % R].cache, knew[j % R], vnew[j % R],
                                                               wls[j % R].Dk, wls[j % R].Dv), K)
    app_ms = time_graph(torch, app_graph, stream) / K
    del dec_graph, app_graph

    # ---- end to end through the public API from pinned host buffers: every
    # step copies its inputs (k_new, v_new, q: one pinned buffer per step) to
    # the device on one copy stream, runs dar_decode_step on the compute stream,
    # and copies its output back on another copy stream; two device input/output
    # buffers let step j's copies overlap step j-1's kernels.  The K steps are
    # one CUDA graph (copies included) replayed once in the timed region.
    nk, nv, nq = knew[0].numel(), vnew[0].numel(), wls[0].q.numel()
    h_in = [torch.cat([knew[j % R].reshape(-1), vnew[j % R].reshape(-1), wls[j % R].q.reshape(-1)]).cpu()
            .pin_memory() for j in range(K)]
    h_out = [torch.empty(outs[0].shape, dtype=outs[0].dtype, pin_memory=True) for _ in range(K)]
    d_in = [torch.empty_like(h_in[0], device=dev) for _ in range(2)]
    d_out = [torch.empty_like(outs[0]) for _ in range(2)]
    views = [(d[:nk].view(knew[0].shape), d[nk:nk + nv].view(vnew[0].shape), d[nk + nv:].view(wls[0].q.shape))
             for d in d_in]
    lens_e2e = [W.download(wl.cache.seq_lens).astype(np.int64) for wl in wls]
    cs_in, cs_out = torch.cuda.Stream(), torch.cuda.Stream()  # host-to-device / device-to-host copies
    e2e = torch.cuda.CUDAGraph()
    with torch.cuda.graph(e2e):
        s = torch.cuda.current_stream()
        fork = torch.cuda.Event()
        fork.record(s)
        cs_in.wait_event(fork)
        cs_out.wait_event(fork)
        done, d2h = [None] * K, [None] * K
        for j in range(K):
            bsel = j % 2
            wl = wls[j % R]
            with torch.cuda.stream(cs_in):
                if j >= 2:
                    cs_in.wait_event(done[j - 2])  # step j-2's kernels have read d_in[bsel]
                d_in[bsel].copy_(h_in[j], non_blocking=True)
                ev_in = torch.cuda.Event()
                ev_in.record(cs_in)
            s.wait_event(ev_in)
            if j >= 2:
                s.wait_event(d2h[j - 2])  # step j-2's output has left d_out[bsel]
            k_c, v_c, q_c = views[bsel]
            dar.dar_decode_step(wl.cache, k_c, v_c, wl.Dk, wl.Dv, q_c, wl.Uk, wl.Uv, wl.workspace, out=d_out[bsel])
            done[j] = torch.cuda.Event()
            done[j].record(s)
            with torch.cuda.stream(cs_out):
                cs_out.wait_event(done[j])
                h_out[j].copy_(d_out[bsel], non_blocking=True)
                d2h[j] = torch.cuda.Event()
                d2h[j].record(cs_out)
        for cs in (cs_in, cs_out):
            join = torch.cuda.Event()
            join.record(cs)
            s.wait_event(join)
    e2e_ms = max_over_ranks(time_graph(torch, e2e, stream), world, dev)
    e2e_bytes = []
    for j in range(K):  # the timed replay is the graph's second: K // R .. steps after lens_e2e
        L_before = lens_e2e[j % R] + len(range(j % R, K, R)) + j // R
        e2e_bytes.append(W.append_step_bytes(cfg, L_before) + W.decode_step_bytes(cfg, L_before + 1))
    e2e_val = world * sum(e2e_bytes) / (e2e_ms * 1e-3) / 1e9
    h2d = h_in[0].numel() * h_in[0].element_size()
    d2h_bytes = outs[0].numel() * outs[0].element_size()
    if sum(wl.cache.device_status() for wl in wls):
        raise RuntimeError("device status set during the end-to-end run")
    del e2e

    prefill = None
    if args.only == "all":
        prefill = prefill_section(args, torch, dar, W, I, dev, stream, tc_peak, peak_src, local)

    extra = None
    # the other workloads and the NEXT rows are measured on single-GPU runs
    # (a multi-GPU run reports the replicated step only, to stay short)
    if args.only == "all" and not args.no_sweep and world == 1:
        del wls, outs, saved, restore, steps_graph
        torch.cuda.empty_cache()
        gqa = decode_only_point(torch, dar, I, W, I.DECODE_1B_GQA, K, l2, dev, stream, hbm_peak)
        sweep = [decode_only_point(torch, dar, I, W, I.sweep_point(k), K, l2, dev, stream, hbm_peak)
                 for k in range(len(I.SWEEP_W) * len(I.SWEEP_DD))]
        direct = {"decode": decode_only_point(torch, dar, I, W, cfg, K, l2, dev, stream, hbm_peak, direct=True),
                  "prefill": direct_prefill_point(args, torch, dar, W, I, dev, stream),
                  "what": "direct lower-dimensional global attention (Sec. 5): dar_attn_decode_direct, "
                          "dar_attn_prefill_direct"}
        extra = {"decode_1b_gqa": gqa, "sweep": sweep, "direct_variant": direct,
                 "backward": backward_point(args, torch, dar, W, I, dev, stream, tc_peak),
                 "latent_form": [latent_point(torch, dar, I, W, c, K, l2, dev, stream, hbm_peak)
                                 for c in (I.DECODE_160M_LATENT, I.DECODE_1B_LATENT)],
                 "note": "graph of K dar_attn_decode calls, rotating cache copies > 4x L2, L2 flushed before"}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        gbs, cores, sample = oracle_decode_sample(cfg, budget_s=args.cpu_budget)
        st_gbs, _, st_sample = oracle_decode_sample(cfg, budget_s=args.cpu_budget / 4, nthreads=1)
        tiny = I.PREFILL_TINY_F32
        x = I.prefill_inputs(tiny)
        t0 = time.perf_counter()
        oracle.prefill(x["q"], x["k"], x["v"], x["Dk"], x["Uk"], x["Dv"], x["Uv"], tiny.w, tiny.dtype, nthreads=1)
        tiny_s = time.perf_counter() - t0
        p_tf, p_cores, p_sample = oracle_prefill_sample(I.PREFILL_410M, budget_s=args.cpu_budget / 3)
        cpu = {"value": round(gbs, 4), "unit": "GB/s", "cores": cores, "kind": "oracle", "sample": sample,
               "single_thread": {
                   "decode-160M": {"value": round(st_gbs, 4), "unit": "GB/s", "cores": 1, "sample": st_sample},
                   "prefill-tiny-f32": {"seconds": round(tiny_s, 4), "cores": 1,
                                        "sample": "the whole workload (4 heads x 256 rows)",
                                        "tflops": round(W.prefill_flops(tiny) / tiny_s / 1e12, 6)}},
               "prefill-410M": {"value": round(p_tf, 6), "unit": "TFLOP/s", "cores": p_cores, "sample": p_sample}}

    if rank == 0:
        line = {
            "metric": METRIC, "value": round(value, 2), "unit": "GB/s", "n_gpus": world, "steps": K, "warmup": Wm,
            "ms_per_step": round(total_ms / K, 5), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic (seeded N(0,1) keys/values/queries)",
            "config": {"workload": cfg.name, "B": cfg.B, "Hq": cfg.Hq, "Hkv": cfg.Hkv, "context": cfg.L,
                       "w": cfg.w, "d": cfg.d, "d_down": cfg.dd, "step": "dar_decode_step: append 1 token + decode",
                       "l2": f"{R} rotating cache copies ({R * one / 1e6:.0f} MB > 4x L2 {l2 / 1e6:.0f} MB), "
                             "restored and L2 flushed before the timed replay",
                       "parallelism": f"{world} independent replicas" if world > 1 else "single GPU"},
            "clocks": clk.summary(),
            "verified": {"oracle_max_abs_err": round(verify_err, 5), "eager_bit_identical": True,
                         "what": "the last timed step of every rotating copy the replay used: sequence 0, all heads"},
            "e2e": {"value": round(e2e_val, 2), "unit": "GB/s", "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h_bytes,
                    "how": "graph of K steps: pinned H2D of k_new,v_new,q -> dar_decode_step -> D2H of out, "
                           "copies on two copy streams overlapping the neighbouring steps' kernels"},
            "gpu_launches": LAUNCHES_PER_STEP * K,
            "roofline": {"bound": "hbm", "achieved": round(dec_gbs, 1), "peak": hbm_peak, "unit": "GB/s",
                         "frac": round(dec_gbs / hbm_peak, 4), "traffic": DECODE_TRAFFIC_BYTES,
                         "kernel": "dar_attn_decode (decode_prep_kernel + decode_kernel<bf16,16,1>)",
                         "bytes_per_launch": int(np.mean(dec_bytes)),
                         "us_per_launch": round(1e3 * dec_ms, 3),
                         "frac_nominal": round(dec_gbs / NOMINAL_HBM_GBS, 4),
                         "peak_source": f"{peak_src} HBM copy"},
            "append_us_per_launch": round(1e3 * app_ms, 3),
            "prefill": prefill,
            "decode_workloads": extra,
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
    ap.add_argument("--no-sweep", action="store_true", help="skip the GQA and sweep decode workloads")
    ap.add_argument("--only", choices=["all", "decode", "prefill", "latent"], default="all",
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
