#!/usr/bin/env python
"""Benchmark of libxhc: connection-op tokens/s, forward + backward, on one GB300 per rank.

One step = the whole hot path over one batch: pre_fwd/post_fwd of every slot of one connection
op group, then post_bwd/pre_bwd of every slot in reverse, on synthetic inputs already resident in
HBM (the state alone is larger than L2, so no L2 flush is needed between steps).  The default
workload is the xHC-Flash-4sub group (slots Attention, MLP, Attention, MLP) with N=16 streams,
k=4 active, m=2 fixed, C=4096, T=32768 tokens (8 sequences of 4096).

Prints one JSON line (rank 0).  ``--impl reference`` times the fp64 CPU oracle instead, on a
bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import hashlib
import glob
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "connection-op tokens/s fwd+bwd at N=16,k=4; achieved HBM GB/s vs peak"


def workloads():
    from paper_2607_14530_gb300.xhc import Config
    return {
        "flash4": ("xHC-Flash-4sub group (A,M,A,M) N=16 k=4 m=2 C=4096 T=32768 (8 x 4096), fwd+bwd",
                   Config.flash(16, 4, 2, 4096, 4, seq_len=4096), 32768),
        "mhc": ("mHC N=4 C=2048 T=8192, fwd+bwd", Config.mhc(4, 2048, seq_len=8192), 8192),
        "fullM": ("full xHC MLP sublayer N=16 k=4 m=2 C=2048 T=16384 (2 x 8192) with TFA, fwd+bwd",
                  Config.full(16, 4, 2, 2048, True, seq_len=8192), 16384),
        "flash4_N4": ("xHC-Flash-4sub N=4 k=4 m=2 C=4096 T=16384, fwd+bwd",
                      Config.flash(4, 4, 2, 4096, 4, seq_len=8192), 16384),
        "flash4_N8": ("xHC-Flash-4sub N=8 k=4 m=2 C=4096 T=16384, fwd+bwd",
                      Config.flash(8, 4, 2, 4096, 4, seq_len=8192), 16384),
        "flash4_N16": ("xHC-Flash-4sub N=16 k=4 m=2 C=4096 T=16384, fwd+bwd",
                       Config.flash(16, 4, 2, 4096, 4, seq_len=8192), 16384),
        "flash4_N32": ("xHC-Flash-4sub N=32 k=4 m=2 C=4096 T=16384, fwd+bwd",
                       Config.flash(32, 4, 2, 4096, 4, seq_len=8192), 16384),
    }


# ---------------------------------------------------------------------------------------------
# algorithmic work of every library launch of one step (bytes each kernel must move at least:
# every input read once, every output written once; flops of the contractions)


# side-stream kernels forked at the same point as a main-stream kernel and overlapping it
OVERLAP = {}
# side-stream kernels whose event window spans main-chain kernels running beside them (the window
# is not the kernel's own duration): not candidates for the dominant kernel
WINDOWED = ("wgrad_tc_full", "wgrad_tc_active")


def kernel_model(cfg, T):
    N, k, C, G = cfg.N, cfg.k, cfg.C, cfg.G
    hr = cfg.m < cfg.k
    nfull = (N if hr else 0) + G * N
    Ks = [cfg.K(t) for t in range(G)]
    nact = [k * Ks[t] + (k * k if t == G - 1 else 0) for t in range(G)]
    S = cfg.seq_len if cfg.seq_len > 0 else T
    gs = cfg.gram_schmidt
    b16, f32 = 2, 4
    m = {}

    def add(name, bytes_=0.0, flops=0.0, bound="hbm"):
        e = m.setdefault(name, dict(launches=0, bytes=0.0, flops=0.0, bound=bound))
        e["launches"] += 1
        e["bytes"] += bytes_
        e["flops"] += flops

    X = T * N * C * b16
    xa = T * k * C * b16
    xa32 = T * k * C * f32
    row = T * C * b16
    kw = max(cfg.conv_k) if cfg.conv_k else 0
    kw = 0 if kw == 0 else (4 if kw <= 4 else 8 if kw <= 8 else 12 if kw <= 12 else 16)
    tb = 296 if kw else 0  # tokens per run of the backward apply (bapp_run)
    runs = (T // S) * -(-S // tb) + -(-(T % S) // tb) if kw else 0
    cpart = runs * sum(cfg.conv_k) * C * f32
    # forward
    if hr:
        add("colsum", N * C * N * f32)
    nb = 2 * nfull  # hi + lo bf16 rows of the packed weight
    add("pack_w", N * C * nfull * f32 + nb * N * C * b16)
    # tensor-core projection: X read once; the packed weight streams from L2
    add("proj_tc", X + T * nfull * f32, 2.0 * T * N * C * nb, "hbm")
    add("coef_full", T * nfull * f32 + T * (G * N + 2 * k) * f32)
    add("read", X + row + (G - 1) * row + xa)
    for t in range(G):
        if t > 0:
            add("input", row + xa + row)
        add("pack_w", k * C * nact[t] * f32 + 2 * nact[t] * k * C * b16)
        add("proj_tc_active", xa + T * nact[t] * f32, 2.0 * T * k * C * 2 * nact[t], "hbm")
        add("coef_act", T * nact[t] * f32 * 2)
        if Ks[t] > 1 and gs:
            add("wb_gram", row)
        add("wb_fwd", row + xa + xa)
    # backward
    for t in reversed(range(G)):
        last = t == G - 1
        dxn = xa if last else xa32
        if last:
            add("restore", 2 * xa)
        if Ks[t] == 1:
            # one pass: out, dXn (and x_act on the last slot) read; d_out and, on the last slot,
            # the mixed active gradient written
            add("wb_b8", row + dxn + (xa if last else 0) + row + (xa32 if last else 0))
        else:
            add("wb_bred", row + dxn + (xa if last else 0))
        add("bwd_coef", T * nact[t] * f32 * 2)
        if Ks[t] > 1:
            # out, dXn read; d_out written; last slot writes the mixed active gradient; conv partials
            add("wb_bapp", row + dxn + row + (xa32 if last else 0) + cpart)
        add("wgrad_tc_active", xa + T * nact[t] * f32 + 2 * T * nact[t] * b16 + k * C * nact[t] * f32,
            2.0 * T * k * C * 2 * nact[t], "hbm")
        add("wgrad_reduce", 2 * k * C * nact[t] * f32)
        for _ in range(4 if last else 2):
            add("colsum", T * 16 * f32)
        if Ks[t] > 1:
            add("conv_wgrad_reduce", cpart)
        # pre-map backward of the slot on the tensor cores: dX_act += dZ W^T + H_pre d_input
        # - cx x_act, with the dH_pre dot partials (per 32 channels) and the d_input copy written in
        # the same pass; then the partials summed per token and active stream
        dotp = k * (C // 32) * T * f32
        add("dxa_tc", 2 * xa32 + xa + row + row + dotp + 3 * T * nact[t] * b16,
            2.0 * T * k * C * 3 * nact[t], "hbm")
        add("dots_act", dotp + T * k * 4 + T * k * f32)
    if hr:
        add("colsum", N * C * N * f32)
    # dH_pre of the inactive streams: their X rows and the G d_input rows read
    add("full_dots", T * (N - k) * C * b16 + G * row)
    add("full_coef", T * (nfull + G * N) * f32)
    # tensor-core dX: X read, inactive dX rows read, active-row gradient read, the G d_input rows
    # read once per column block (dense-read gradient of the inactive rows), dX written
    add("dx_tc", X + T * (N - k) * C * b16 + xa32 + G * row + X, 2.0 * T * N * C * nfull, "hbm")
    add("wgrad_tc_full", X + T * nfull * f32 + 2 * T * nfull * b16 + N * C * nfull * f32,
        2.0 * T * N * C * 2 * nfull, "hbm")
    add("wgrad_reduce", 2 * N * C * nfull * f32)
    add("colsum", T * G * N * f32)
    add("colsum", T * G * f32)
    if hr:
        add("colsum", T * N * f32)
        add("sub_rows", 2 * N * C * N * f32)
    return m


def paper_forward_bytes_per_token(cfg):
    """Forward traffic of Table overhead_analysis for this group, bytes per token."""
    from paper_2607_14530_gb300 import traffic
    return traffic.forward_model("mhc" if cfg.variant == 0 else "xhc", cfg.N, cfg.k, cfg.G) * cfg.C * 2


def model_bytes_per_token(cfg):
    """(forward, backward) algorithmic bytes per token of one group: the paper's forward
    accounting and the backward model of traffic.backward_model (bf16 = 2 bytes)."""
    from paper_2607_14530_gb300 import traffic
    return paper_forward_bytes_per_token(cfg), traffic.backward_model(cfg.N, cfg.k, cfg.G) * cfg.C * 2


# ---------------------------------------------------------------------------------------------
# clocks during the timed region


class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, dev: int):
        self.dev = dev
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200", "-i", str(self.dev)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except OSError:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.t.join(timeout=2)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            p = [x.strip() for x in ln.split(",")]
            if len(p) < 8:
                continue
            try:
                sm.append(float(p[0]))
                mx.append(float(p[1]))
            except ValueError:
                continue
            for nm, v in zip(names, p[4:8]):
                if v.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "reasons": sorted(reasons)}


# ---------------------------------------------------------------------------------------------


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "sm_max_mhz": 2070.0}, "fallback"


def csrc_hash():
    h = hashlib.sha256()
    for f in sorted(glob.glob(os.path.join(ROOT, "paper_2607_14530_gb300", "csrc", "*"))):
        with open(f, "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def ncu_traffic(kernel, workload):
    """DRAM bytes per launch from the committed ncu summary, if it was taken on the current
    kernel sources and this workload; else None."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    e = d.get(workload, {}).get(kernel)
    if not e or e.get("csrc_sha") != csrc_hash():
        return None
    return e.get("dram_bytes_per_launch")


def ncu_forward_bytes(workload):
    """Measured forward DRAM bytes per token (ncu, the forward kernels of one group) from the
    committed summary, if it was taken on the current kernel sources; else None."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    e = d.get(workload, {}).get("_forward")
    if not e or e.get("csrc_sha") != csrc_hash():
        return None
    return e.get("dram_bytes_per_token")


def job_rate(ms_local, tokens_per_rank, steps, world, device=None):
    """(slowest rank's ms, whole-job tokens/s): every rank processes its own tokens_per_rank per
    step (weak scaling, no data-path collective); the timed region is the max over ranks."""
    ms = float(ms_local)
    if world > 1:
        import torch
        import torch.distributed as dist
        t = torch.tensor([ms], dtype=torch.float64, device=device)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = float(t.item())
    return ms, world * tokens_per_rank * steps / (ms / 1000.0)


def oracle_step(cfg, X, outs, dX, dins, P):
    """One fp64 oracle fwd+bwd on CPU tensors (the oracle as it stands)."""
    import torch
    from oracle import xhc_oracle as O
    ocfg = O.Config(N=cfg.N, k=cfg.k, m=cfg.m, C=cfg.C, G=cfg.G,
                    mlp=tuple(bool((cfg.mlp_mask >> t) & 1) for t in range(cfg.G)),
                    conv_k=tuple(cfg.conv_k), gram_schmidt=cfg.gram_schmidt,
                    sinkhorn_iters=cfg.sinkhorn_iters, eps_norm=cfg.eps_norm,
                    eps_gs=(cfg.eps_gs if cfg.eps_gs > 0 else None), seq_len=cfg.seq_len,
                    router=cfg.router, dense_read=not cfg.sparse_read)
    f64 = torch.float64
    P64 = {n: v.to(f64) for n, v in P.items()}
    O.backward(ocfg, P64, X.to(f64), [o.to(f64) for o in outs], dX.to(f64), [d.to(f64) for d in dins])


def cpu_sample(cfg, T_s, seed):
    import torch
    from paper_2607_14530_gb300 import synth
    d = synth.group_inputs(T_s, cfg.N, cfg.C, cfg.G, seed)
    g = synth.group_grads(T_s, cfg.N, cfg.C, cfg.G, seed)
    P = synth.params(cfg.param_shapes(), seed)
    return d["X"], d["outs"], g["dX"], g["d_inputs"], P


def run_reference(args, wl_name):
    import torch
    desc, cfg, T = workloads()[wl_name]
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    T_s = args.ref_tokens
    X, outs, dX, dins, P = cpu_sample(cfg, T_s, 0)
    for _ in range(args.warmup):
        oracle_step(cfg, X, outs, dX, dins, P)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle_step(cfg, X, outs, dX, dins, P)
    dt = time.perf_counter() - t0
    value = T_s * args.steps / dt
    cores = torch.get_num_threads()
    sample = f"first {T_s} tokens of sequence 0 of the workload per step (fp64 oracle, fwd+bwd)"
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1000.0 * dt / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": desc, "tokens_per_step": T_s},
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_xhc(args, wl_name):
    import torch
    import torch.distributed as dist
    from paper_2607_14530_gb300 import build, synth, xhc

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)
    if rank == 0:
        build.build()
    if world > 1:
        dist.barrier()
    xhc.lib()

    desc, cfg, T = workloads()[wl_name]
    if args.tokens:
        T = args.tokens
    g = xhc.Group(cfg)
    seed = 1234 + rank
    X = synth.normal_bf16_on((T, cfg.N, cfg.C), seed, dev)
    outs = [synth.normal_bf16_on((T, cfg.C), seed + 101 + t, dev) for t in range(cfg.G)]
    dX0 = synth.normal_bf16_on((T, cfg.N, cfg.C), seed + 7, dev)
    dins = [synth.normal_bf16_on((T, cfg.C), seed + 211 + t, dev) for t in range(cfg.G)]
    P = {n: v.to(dev) for n, v in synth.params(cfg.param_shapes(), seed).items()}
    G_ = {n: torch.zeros_like(v) for n, v in P.items()}
    saved, ws = g.alloc(T, device=dev)
    inputs = [torch.empty(T, cfg.C, dtype=torch.bfloat16, device=dev) for _ in range(cfg.G)]
    d_outs = [torch.empty(T, cfg.C, dtype=torch.bfloat16, device=dev) for _ in range(cfg.G)]
    dX = dX0.clone()
    stream = torch.cuda.current_stream()

    def step():
        g.forward(P, X, outs, saved, ws, inputs=inputs)
        g.backward(P, X, dX, outs, dins, G_, saved, ws, d_outs=d_outs)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()

    # per-kernel device times: a traced pass of the same steps before the timed region (events
    # around every launch cost the step about 0.3 ms, so the timed region records only the
    # dominant kernel and the side-stream kernels that share its window)
    model = kernel_model(cfg, T)
    xhc.trace_only(None)
    xhc.trace_enable(True)
    for _ in range(args.steps):
        step()
    torch.cuda.synchronize()
    xhc.trace_enable(False)
    recs = xhc.trace_spans()
    per = {}
    for name, _t0, t_ms in recs:
        e = per.setdefault(name, [0, 0.0])
        e[0] += 1
        e[1] += t_ms
    dom = max((n for n in per if n in model and n not in WINDOWED), key=lambda n: per[n][1])

    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    xhc.trace_only((dom,) + tuple(OVERLAP.get(dom, ())))
    xhc.trace_enable(True)
    n0 = xhc.launch_count()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    launches = xhc.launch_count() - n0
    xhc.trace_enable(False)
    xhc.trace_only(None)
    ck = clocks.stop()
    ms, value = job_rate(e0.elapsed_time(e1), T, args.steps, world, dev)
    ms_step = ms / args.steps

    # the dominant kernel and its window partners over the timed region
    live = {}
    for name, t_ms in xhc.trace_records():
        e = live.setdefault(name, [0, 0.0])
        e[0] += 1
        e[1] += t_ms
    peaks, peak_src = measured_peaks()
    hbm_peak = float(peaks["hbm_gbs"])
    sm_mhz = float(peaks.get("sm_max_mhz", 2070.0))
    alu_peak = 152 * 128 * 2 * sm_mhz * 1e6 / 1e12  # fp32 FMA lanes x 2 flop x max clock, TFLOP/s
    kernels = {}
    for name, (cnt, tot) in per.items():
        mm = model.get(name)
        ent = {"launches": cnt // args.steps, "ms_per_step": tot / args.steps,
               "share": tot / max(1e-9, sum(v[1] for v in per.values()))}
        if mm:
            secs = tot / args.steps / 1000.0
            ent["gbs"] = mm["bytes"] / secs / 1e9
            if mm["flops"]:
                ent["tflops"] = mm["flops"] / secs / 1e12
            ent["bound"] = mm["bound"]
        kernels[name] = ent
    mm = model[dom]
    cnt, tot = live[dom]
    secs = tot / cnt / 1000.0
    launches_per_step = mm["launches"]
    if mm["bound"] == "alu":
        achieved = mm["flops"] / launches_per_step / secs / 1e12
        roof = {"kernel": dom, "bound": "alu", "achieved": achieved, "peak": alu_peak,
                "unit": "TFLOP/s", "frac": achieved / alu_peak,
                "peak_source": "derived: 152 SMs x 128 fp32 lanes x 2 flop x max SM clock"}
    else:
        achieved = mm["bytes"] / launches_per_step / secs / 1e9
        roof = {"kernel": dom, "bound": "hbm", "achieved": achieved, "peak": hbm_peak,
                "unit": "GB/s", "frac": achieved / hbm_peak, "peak_source": f"{peak_src} hbm_gbs"}
    roof["traffic"] = ncu_traffic(dom, wl_name)
    # kernels the library launches on its side stream at the same point, which finish inside the
    # dominant kernel's event window and share its HBM bandwidth: their bytes over that window
    part = [n for n in OVERLAP.get(dom, ()) if n in live and n in model and live[n][1] <= tot]
    if part and roof["bound"] == "hbm":
        wb = mm["bytes"] / launches_per_step + sum(model[n]["bytes"] / model[n]["launches"] for n in part)
        roof["concurrent"] = {"kernels": part, "window_gbs": wb / secs / 1e9,
                              "window_frac": wb / secs / 1e9 / hbm_peak,
                              "note": "side-stream kernels running inside this kernel's launch window; "
                                      "achieved / frac above count this kernel's bytes only"}

    step_bytes = sum(v["bytes"] for v in model.values())
    fb, bb = model_bytes_per_token(cfg)
    alg = (fb + bb) * T
    hbm = {"kernel_model_bytes_per_step": step_bytes,
           "kernel_model_gbs": step_bytes / (ms_step / 1000.0) / 1e9,
           "kernel_model_frac": step_bytes / (ms_step / 1000.0) / 1e9 / hbm_peak,
           "algorithmic_bytes_per_step": alg,
           "algorithmic_gbs": alg / (ms_step / 1000.0) / 1e9,
           "algorithmic_frac": alg / (ms_step / 1000.0) / 1e9 / hbm_peak,
           "algorithmic_model": "paper forward accounting (Table overhead_analysis) + traffic.backward_model, "
                                "bf16, per group per token: fwd %.0f B + bwd %.0f B" % (fb, bb),
           "paper_fwd_bytes_per_token": fb}

    # forward only (prefill-style: pre_fwd / post_fwd of every slot), same inputs, CUDA events
    def fwd_step():
        g.forward(P, X, outs, saved, ws, inputs=inputs)

    for _ in range(2):
        fwd_step()
    torch.cuda.synchronize()
    f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    f0.record(stream)
    for _ in range(args.steps):
        fwd_step()
    f1.record(stream)
    torch.cuda.synchronize()
    fms, fvalue = job_rate(f0.elapsed_time(f1), T, args.steps, world, dev)
    fwd = {"tokens_per_s": fvalue, "ms_per_step": fms / args.steps,
           "algorithmic_frac": fb * T / (fms / args.steps / 1000.0) / 1e9 / hbm_peak}
    dram = ncu_forward_bytes(wl_name)
    if dram is not None:
        fwd["dram_bytes_per_token"] = dram
        fwd["dram_vs_paper_model"] = dram / fb
        fwd["gate"] = "<= 1.2 x the paper's forward model"

    line = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic",
            "config": {"workload": desc, "tokens": T, "storage": "bf16 state, fp32 params/coefficients",
                       "l2": "inputs larger than L2 (state alone is %.1f GiB), no flush" % (T * cfg.N * cfg.C * 2 / 2**30),
                       "parallelism": "replicas" if world > 1 else "1 GPU"},
            "roofline": roof, "hbm": hbm, "fwd": fwd, "gpu_launches": launches, "clocks": ck}

    if args.kernels_out and rank == 0:
        with open(args.kernels_out, "w") as f:
            one = recs[:len(recs) // max(1, args.steps)]
            seq = [[n, t_ms, t0 - one[0][1]] for n, t0, t_ms in one]
            json.dump({"workload": wl_name, "kernels": kernels, "model": model, "sequence": seq}, f,
                      indent=1)

    # end to end through the public API with host buffers: every step copies its inputs host ->
    # device from pinned memory, runs, and copies its results device -> host.  Steps are
    # pipelined the way a caller would run them: two device buffer sets, inputs of step i+1
    # copied in (copy-in stream) while step i computes, results of step i copied out (copy-out
    # stream) while step i+1 computes.  The timed region runs from the first copy-in to the last
    # copy-out.
    if not args.no_e2e:
        pin = lambda t: torch.empty(t.shape, dtype=t.dtype, pin_memory=True)  # noqa: E731
        hX, hdX = pin(X), pin(dX)
        hX.copy_(X)
        hdX.copy_(dX0)
        houts = [pin(o) for o in outs]
        hdins = [pin(d) for d in dins]
        for h, d in zip(houts + hdins, outs + dins):
            h.copy_(d)
        rdX = pin(dX)
        rins = [pin(i) for i in inputs]
        rdouts = [pin(o) for o in d_outs]
        h2d = sum(t.numel() * t.element_size() for t in [hX, hdX] + houts + hdins)
        d2h = sum(t.numel() * t.element_size() for t in [rdX] + rins + rdouts)
        sets = [dict(X=X, dX=dX, outs=outs, dins=dins, inputs=inputs, d_outs=d_outs)]
        sets.append(dict(X=torch.empty_like(X), dX=torch.empty_like(dX),
                         outs=[torch.empty_like(o) for o in outs], dins=[torch.empty_like(d) for d in dins],
                         inputs=[torch.empty_like(i) for i in inputs], d_outs=[torch.empty_like(o) for o in d_outs]))
        s_in, s_out = torch.cuda.Stream(), torch.cuda.Stream()
        ev_in = [torch.cuda.Event() for _ in range(2)]
        ev_comp = [torch.cuda.Event() for _ in range(2)]
        ev_out = [torch.cuda.Event() for _ in range(2)]

        def copy_in(b):
            with torch.cuda.stream(s_in):
                s_in.wait_event(ev_out[b])     # the set's previous results are out
                sb = sets[b]
                sb["X"].copy_(hX, non_blocking=True)
                sb["dX"].copy_(hdX, non_blocking=True)
                for d, h in zip(sb["outs"] + sb["dins"], houts + hdins):
                    d.copy_(h, non_blocking=True)
                ev_in[b].record(s_in)

        def compute(b):
            stream.wait_event(ev_in[b])
            sb = sets[b]
            g.forward(P, sb["X"], sb["outs"], saved, ws, inputs=sb["inputs"], stream=stream)
            g.backward(P, sb["X"], sb["dX"], sb["outs"], sb["dins"], G_, saved, ws, d_outs=sb["d_outs"],
                       stream=stream)
            ev_comp[b].record(stream)

        def copy_out(b):
            with torch.cuda.stream(s_out):
                s_out.wait_event(ev_comp[b])
                sb = sets[b]
                rdX.copy_(sb["dX"], non_blocking=True)
                for h, d in zip(rins + rdouts, sb["inputs"] + sb["d_outs"]):
                    h.copy_(d, non_blocking=True)
                ev_out[b].record(s_out)

        def run(n, a=None, z=None):
            for ev in ev_out:
                ev.record(s_out)
            if a is not None:
                a.record(s_in)
            copy_in(0)
            for i in range(n):
                if i + 1 < n:
                    copy_in((i + 1) % 2)
                compute(i % 2)
                copy_out(i % 2)
            if z is not None:
                z.record(s_out)

        ksteps = max(2, min(args.steps, 5))
        run(2)
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        run(ksteps, a, b)
        torch.cuda.synchronize()
        ems, evalue = job_rate(a.elapsed_time(b), T, ksteps, world, dev)
        line["e2e"] = {"value": evalue, "unit": "tokens/s",
                       "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": ksteps,
                       "pipelined": "copy-in of step i+1 and copy-out of step i overlap step i+1's compute"}

    # inference leg: decode steps of the same group shape (B sequences, one new token each)
    if not args.no_decode:
        line["decode"] = decode_leg(cfg, P, args.decode_batch, max(5, args.steps), dev, stream)

    if rank == 0 and not args.no_cpu_baseline:
        T_s = args.cpu_tokens
        Xs, os_, dXs, dis, Ps = cpu_sample(cfg, T_s, 0)
        t0 = time.perf_counter()
        oracle_step(cfg, Xs, os_, dXs, dis, Ps)
        dt = time.perf_counter() - t0
        line["cpu_baseline"] = {"value": T_s / dt, "unit": "tokens/s", "cores": torch.get_num_threads(),
                                "kind": "oracle",
                                "sample": f"first {T_s} tokens of one sequence of the workload, fp64 "
                                          f"oracle fwd+bwd, one run of {dt:.1f} s"}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def decode_leg(cfg, P, B, steps, dev, stream, seed=1234):
    """Decode steps of one group (one new token for each of B sequences, conv history in rings,
    positions past 4096), eagerly and replayed as a captured CUDA graph of one step; CUDA events
    on the launching stream."""
    import torch
    from paper_2607_14530_gb300 import synth, xhc

    def timed(fn, k):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(k):
            fn()
        b.record(stream)
        torch.cuda.synchronize()
        return a.elapsed_time(b) / k

    gd = xhc.Group(type(cfg).flash(cfg.N, cfg.k, cfg.m, cfg.C, cfg.G, seq_len=0) if cfg.G > 1 else cfg)
    Xd = synth.normal_bf16_on((B, cfg.N, cfg.C), seed + 3, dev)
    outs_d = [synth.normal_bf16_on((B, cfg.C), seed + 301 + t, dev) for t in range(cfg.G)]
    saved_d, ws_d = gd.alloc(B, device=dev)
    rings = gd.alloc_rings(B, device=dev)
    pos = torch.full((B,), 4096, dtype=torch.int64, device=dev)
    ins_d = [torch.empty(B, cfg.C, dtype=torch.bfloat16, device=dev) for _ in range(cfg.G)]

    def dstep():
        gd.forward_decode(P, Xd, outs_d, rings, pos, saved_d, ws_d, inputs=ins_d)

    eager_ms = timed(dstep, steps)
    n0 = xhc.launch_count()
    xhc.trace_enable(True)
    dstep()
    torch.cuda.synchronize()
    launches = xhc.launch_count() - n0
    per = {}
    for name, t_ms in xhc.trace_records():
        per[name] = per.get(name, 0.0) + t_ms
    xhc.trace_enable(False)
    top = sorted(per.items(), key=lambda kv: -kv[1])[:6]
    graph_ms = None
    try:
        graph = torch.cuda.CUDAGraph()
        side = torch.cuda.Stream()
        side.wait_stream(stream)
        with torch.cuda.stream(side):
            dstep()
        stream.wait_stream(side)
        torch.cuda.synchronize()
        with torch.cuda.graph(graph):
            dstep()
        graph_ms = timed(graph.replay, steps)
    except Exception as e:  # capture not possible on this stack: eager numbers only
        graph_ms = f"not captured: {type(e).__name__}"
    return {"batch": B, "launches_per_step": launches, "eager_ms": eager_ms,
            "top_calls_ms": [[n, round(t, 4)] for n, t in top],
            "eager_value": B / (eager_ms / 1000.0), "graph_ms": graph_ms,
            "graph_value": (B / (graph_ms / 1000.0)) if isinstance(graph_ms, float) else None,
            "unit": "tokens/s", "note": "one group of G sublayers per token"}


def run_decode(args, wl_name):
    """Inference legs (not part of the default line): forward-only prefill of the workload, and
    decode steps (one new token per sequence, conv history in rings) for a batch of sequences,
    eagerly and as a captured CUDA graph of one step.  One JSON line."""
    import torch
    from paper_2607_14530_gb300 import build, synth, xhc

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    build.build()
    xhc.lib()
    desc, cfg, T = workloads()[wl_name]
    if args.tokens:
        T = args.tokens
    seed = 1234
    P = {n: v.to(dev) for n, v in synth.params(cfg.param_shapes(), seed).items()}
    stream = torch.cuda.current_stream()

    def timed(fn, k):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(k):
            fn()
        b.record(stream)
        torch.cuda.synchronize()
        return a.elapsed_time(b) / k

    # prefill: the forward of the whole workload (sequences of seq_len tokens)
    g = xhc.Group(cfg)
    X = synth.normal_bf16_on((T, cfg.N, cfg.C), seed, dev)
    outs = [synth.normal_bf16_on((T, cfg.C), seed + 101 + t, dev) for t in range(cfg.G)]
    saved, ws = g.alloc(T, device=dev)
    inputs = [torch.empty(T, cfg.C, dtype=torch.bfloat16, device=dev) for _ in range(cfg.G)]
    X0 = X.clone()

    def prefill():
        X.copy_(X0)
        g.forward(P, X, outs, saved, ws, inputs=inputs)

    copy_ms = timed(lambda: X.copy_(X0), args.steps)
    pre_ms = timed(prefill, args.steps) - copy_ms
    del saved, ws, X, X0, inputs
    torch.cuda.empty_cache()

    dec = decode_leg(cfg, P, args.decode_batch, args.steps, dev, stream, seed)
    line = {"metric": "inference: prefill and decode tokens/s", "unit": "tokens/s",
            "prefill": {"workload": desc, "tokens": T, "ms": pre_ms, "value": T / (pre_ms / 1000.0)},
            "decode": dec,
            "steps": args.steps, "dtype": "f32", "data": "synthetic"}
    print(json.dumps(line), flush=True)


def run_stack(args, wl_name):
    """A stack of L groups through the model glue (stream expansion, L groups of the workload's
    shape with scalar-gain sublayers, final stream sum; forward and torch.autograd backward),
    against L bare group calls (forward + backward through the binding) on the same tokens: the
    glue's overhead.  One JSON line; CUDA events on the current stream."""
    import torch
    from torch import nn
    from paper_2607_14530_gb300 import build, synth, xhc
    from paper_2607_14530_gb300.model import XhcStack

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    build.build()
    xhc.lib()
    desc, cfg, T = workloads()[wl_name]
    T = args.tokens or 8192
    L = args.groups
    seed = 1234

    class Gain(nn.Module):
        def __init__(self):
            super().__init__()
            self.s = nn.Parameter(torch.tensor(0.03125))

        def forward(self, x):
            return x * self.s.to(x.dtype)

    stack = XhcStack(cfg, L, lambda l, t: Gain(), seed=seed).to(dev)
    hid = synth.normal_bf16_on((T, cfg.C), seed + 5, dev)
    dy = synth.normal_bf16_on((T, cfg.C), seed + 6, dev)
    stream = torch.cuda.current_stream()

    def stack_step():
        h = hid.detach().requires_grad_(True)
        y = stack(h)
        y.backward(dy)

    def timed(fn, k):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(k):
            fn()
        b.record(stream)
        torch.cuda.synchronize()
        return a.elapsed_time(b) / k

    stack_ms = timed(stack_step, args.steps)
    # the same work as bare group calls: L x (forward + backward of one group)
    g = xhc.Group(cfg)
    P = {n: v.to(dev) for n, v in synth.params(cfg.param_shapes(), seed).items()}
    G_ = {n: torch.zeros_like(v) for n, v in P.items()}
    saved, ws = g.alloc(T, device=dev)
    X = synth.normal_bf16_on((T, cfg.N, cfg.C), seed, dev)
    outs = [synth.normal_bf16_on((T, cfg.C), seed + 101 + t, dev) for t in range(cfg.G)]
    dX = synth.normal_bf16_on((T, cfg.N, cfg.C), seed + 7, dev)
    dins = [synth.normal_bf16_on((T, cfg.C), seed + 211 + t, dev) for t in range(cfg.G)]
    inputs = [torch.empty(T, cfg.C, dtype=torch.bfloat16, device=dev) for _ in range(cfg.G)]
    d_outs = [torch.empty(T, cfg.C, dtype=torch.bfloat16, device=dev) for _ in range(cfg.G)]

    def bare_step():
        for _ in range(L):
            g.forward(P, X, outs, saved, ws, inputs=inputs)
            g.backward(P, X, dX, outs, dins, G_, saved, ws, d_outs=d_outs)

    bare_ms = timed(bare_step, args.steps)
    # the parts of a stack step that are neither the library's group calls nor glue: the L x G
    # sublayers' own forward and backward, and the stream expansion and sum with their backward
    gains = [Gain().to(dev) for _ in range(L * cfg.G)]

    def sublayer_step():
        for m in gains:
            x = hid.detach().requires_grad_(True)
            m(x).backward(hid)

    sub_ms = timed(sublayer_step, args.steps)
    gx = stack.groups[0].g

    def expand_sum_step():
        Xs = gx.stream_expand(hid)
        gx.stream_sum(Xs)
        gx.stream_expand(dy)
        gx.stream_sum(Xs)

    es_ms = timed(expand_sum_step, args.steps)
    line = {"metric": "stack of groups through the autograd glue: tokens/s fwd+bwd", "unit": "tokens/s",
            "workload": f"{L} groups of: {desc}; sublayers: scalar gains (bf16)", "tokens": T,
            "stack_ms": stack_ms, "value": T / (stack_ms / 1000.0),
            "bare_group_calls_ms": bare_ms, "sublayers_ms": sub_ms, "expand_sum_ms": es_ms,
            "glue_overhead": (stack_ms - sub_ms - es_ms) / bare_ms - 1.0,
            "note": "glue_overhead: the stack step less the sublayers' own work and the stream "
                    "expansion / sum, over the bare group calls, minus 1",
            "steps": args.steps, "dtype": "f32", "data": "synthetic"}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="xhc", choices=["xhc", "reference"])
    ap.add_argument("--workload", default="flash4")
    ap.add_argument("--tokens", type=int, default=0, help="override T (development only)")
    ap.add_argument("--cpu-tokens", type=int, default=3072)
    ap.add_argument("--ref-tokens", type=int, default=64)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-decode", action="store_true", help="skip the decode leg of the default line")
    ap.add_argument("--kernels-out", default="")
    ap.add_argument("--mode", default="train", choices=["train", "inference", "stack"],
                    help="inference: forward-only prefill and decode legs; stack: a stack of groups "
                         "through the autograd glue (separate lines)")
    ap.add_argument("--groups", type=int, default=4, help="groups of the stack leg")
    ap.add_argument("--decode-batch", type=int, default=256)
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "xhc":
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args, args.workload)
    elif args.mode == "inference":
        run_decode(args, args.workload)
    elif args.mode == "stack":
        run_stack(args, args.workload)
    else:
        run_xhc(args, args.workload)


if __name__ == "__main__":
    main()
