"""Benchmark of the MoE-ViE fine-grained MoE FFN layer forward on GB300.

One step = one whole layer forward (router, expert-major order, grouped up- and
down-projection with the fused combine, shared expert, final bf16 output) over
one batch of synthetic tokens, through the C ABI (moevie_moe_forward).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--config c4] [--extra c1,c2,c3]
                    [--impl ours|reference]

Prints one JSON line.  Default workload: the largest single-GPU layer, the stress
layer (c4: T=65536, d=1664, E=256, k=8, h=416, one saturated expert, Zipf(1.1)
loads over the rest, 3 empty experts).  On one GPU the other layers named by
--extra are measured after it and reported under "per_config" (device-resident
time, layer roofline fraction, stage times, memory-bound stages).  Under torchrun
each rank runs its own replica of the workload (tokens shard with no exchange
step), the timed region is bracketed by barriers, and the slowest rank's time is
used.  `--impl reference` times the CPU oracle on a bounded token sample instead.
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

import workloads  # noqa: E402

METRIC = "MoE-layer tokens/sec and µs/layer on 1 GB300; achieved fraction of roofline"
L2_FLUSH_BYTES = 512 << 20


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--config", default="c4", choices=sorted(workloads.CONFIGS))
    ap.add_argument("--extra", default="c1,c2,c3",
                    help="other workloads measured after the main one (1 GPU only; '' for none)")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-backward", action="store_true", help="skip timing the training path")
    ap.add_argument("--gemm-calibration", action="store_true",
                    help="instead of a layer: the library's dense GEMM pair (moevie_shared_expert: "
                         "x Ws1 with GELU, then . Ws2) against cuBLAS (torch.matmul) on a few shapes, "
                         "one JSON line each")
    return ap.parse_args()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            mp = json.load(f)
        return {"hbm_gbs": float(mp["hbm_gbs"]), "bf16_tflops": float(mp["bf16_tflops"]),
                "bf16_tflops_sustained": float(mp.get("bf16_tflops_sustained", mp["bf16_tflops"])),
                "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
            "source": "fallback"}


GEMM_SOURCES = ("paper_2608_17402_gb300/csrc/gemm.cu", "paper_2608_17402_gb300/csrc/common.cuh",
                "paper_2608_17402_gb300/csrc/internal.h")
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "grouped_gemm_dram_traffic.json")


def gemm_sources_hash():
    import hashlib
    h = hashlib.sha256()
    for rel in GEMM_SOURCES:
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def captured_traffic(cfg_name, stage):
    """DRAM bytes (read + write) of one grouped GEMM launch from the committed ncu
    capture, or None when there is none for this workload or the GEMM sources have
    changed since it was taken."""
    if not os.path.exists(TRAFFIC_FILE):
        return None
    with open(TRAFFIC_FILE) as f:
        rec = json.load(f)
    if rec.get("sources_sha256") != gemm_sources_hash():
        return None
    per = rec.get("workloads", {}).get(cfg_name, {}).get(stage)
    return None if per is None else float(per["dram_bytes"])


def layer_work(cfg, counts, shared_groups=0):
    """Algorithmic FLOPs and bytes of one layer forward (weights of touched experts).
    shared_groups: always-on groups of width h that carry the shared expert inside the
    routed up / down launches (moevie_shared_groups), counted in those launches' FLOPs."""
    T, d, E, k, h, hs = cfg.T, cfg.d, cfg.E, cfg.k, cfg.h, cfg.h_s
    up_mats = 2 if cfg.act == "swiglu" else 1    # SwiGLU: gate (W1) and up (W3) projections
    flops_router = 2.0 * T * d * E
    flops_up = 2.0 * up_mats * T * k * d * h
    flops_down = 2.0 * T * k * d * h
    flops_shared = 2.0 * (up_mats + 1) * T * d * hs
    touched = int((np.asarray(counts) > 0).sum())
    bytes_ = (T * d * 2 + T * d * 2 + d * E * 4 + E * 4 + touched * (up_mats + 1) * d * h * 2
              + (up_mats + 1) * d * hs * 2 + 8 * T * k)
    folded = shared_groups * h * T * d * 2.0
    return {"flops": flops_router + flops_up + flops_down + flops_shared,
            "flops_up_gemm": flops_up + up_mats * folded,
            "flops_down_gemm": flops_down + folded, "bytes": float(bytes_), "touched_experts": touched}


class ClockSampler:
    """nvidia-smi clock / throttle samples during the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = os.path.join("/tmp", f"moevie_clocks_{os.getpid()}.csv")

    def __enter__(self):
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            time.sleep(0.2)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.f.close()

    def summary(self):
        if self.proc is None or not os.path.exists(self.path):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                p = [x.strip() for x in line.split(",")]
                if len(p) < 9:
                    continue
                try:
                    sm.append(float(p[1]))
                    smax.append(float(p[2]))
                except ValueError:
                    continue
                for n, v in zip(names, p[5:9]):
                    if v.lower() == "active":
                        reasons.add(n)
        os.remove(self.path)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        loaded = [s for s in sm if s > 0.5 * max(sm)] or sm
        return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm)}


def cpu_baseline(lay, target_s=15.0, max_tokens=None):
    """The oracle, as it stands, on a bounded token sample (host cores)."""
    import oracle
    cfg = lay.cfg
    nthreads = oracle.default_threads()
    rng = np.random.default_rng(123)
    probe = np.sort(rng.choice(cfg.T, size=min(cfg.T, max(nthreads, 8)), replace=False)).astype(np.int32)
    t0 = time.perf_counter()
    oracle.forward_tokens(lay.x, lay.Wr, lay.b, lay.W1, lay.W2, cfg.k, lay.Ws1, lay.Ws2, cfg.lam, tokens=probe, W3=lay.W3, Ws3=lay.Ws3)
    per_tok = (time.perf_counter() - t0) / probe.size
    n = int(min(cfg.T, max(nthreads, target_s / max(per_tok, 1e-9))))
    if max_tokens:
        n = min(n, max_tokens)
    toks = np.sort(rng.choice(cfg.T, size=n, replace=False)).astype(np.int32)
    # whole passes over the sample until about target_s of CPU time has been spent
    passes, t0 = 0, time.perf_counter()
    while True:
        oracle.forward_tokens(lay.x, lay.Wr, lay.b, lay.W1, lay.W2, cfg.k, lay.Ws1, lay.Ws2, cfg.lam,
                              tokens=toks, W3=lay.W3, Ws3=lay.Ws3)
        passes += 1
        dt = time.perf_counter() - t0
        if dt >= 0.66 * target_s or passes >= 8:
            break
    return {"value": passes * n / dt, "unit": "tokens/s", "cores": nthreads, "kind": "oracle",
            "sample": f"{passes} pass(es) over {n} of {cfg.T} tokens of {cfg.name} (whole layer per "
                      f"token: route, k experts, shared expert), fp64, {nthreads} threads, {dt:.1f} s"}


def run_reference(args, rank):
    if rank != 0:
        return
    cfg = workloads.CONFIGS[args.config]
    lay = workloads.make_layer(cfg)
    import oracle
    nthreads = oracle.default_threads()
    rng = np.random.default_rng(7)
    # size each step so the whole run stays within a few minutes
    probe = np.arange(min(cfg.T, nthreads), dtype=np.int32)
    t0 = time.perf_counter()
    oracle.forward_tokens(lay.x, lay.Wr, lay.b, lay.W1, lay.W2, cfg.k, lay.Ws1, lay.Ws2, cfg.lam, tokens=probe, W3=lay.W3, Ws3=lay.Ws3)
    per_tok = (time.perf_counter() - t0) / probe.size
    budget = 150.0 / max(1, args.steps + args.warmup)
    n = int(min(cfg.T, max(nthreads, budget / max(per_tok, 1e-9))))
    times = []
    for i in range(args.warmup + args.steps):
        toks = np.sort(rng.choice(cfg.T, size=n, replace=False)).astype(np.int32)
        t0 = time.perf_counter()
        oracle.forward_tokens(lay.x, lay.Wr, lay.b, lay.W1, lay.W2, cfg.k, lay.Ws1, lay.Ws2, cfg.lam,
                              tokens=toks, W3=lay.W3, Ws3=lay.Ws3)
        if i >= args.warmup:
            times.append(time.perf_counter() - t0)
    ms = 1e3 * statistics.mean(times)
    value = n / (ms / 1e3)
    out = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": args.gpus,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
           "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "config": {"workload": f"{cfg.name}: {cfg.note}", "T": cfg.T, "d": cfg.d, "E": cfg.E, "k": cfg.k,
                      "h": cfg.h, "h_s": cfg.h_s, "act": cfg.act, "tokens_per_step": n},
           "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": nthreads, "kind": "oracle",
                            "sample": f"{n} random tokens of {cfg.name} per step"},
           "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


def _device_layer(cfg, lay, moevie, torch):
    def bf(a):
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).cuda()

    def rows(a):   # W1, W3, Ws1, Ws3: rows 16 bytes apart (h rounded up to 8)
        return moevie.moevie_pad_rows(bf(a))

    W = moevie.LayerWeights(W_r=torch.from_numpy(lay.Wr).cuda(), b=torch.from_numpy(lay.b).cuda(),
                            W1=rows(lay.W1), W2=bf(lay.W2), k=cfg.k,
                            Ws1=None if lay.Ws1 is None else rows(lay.Ws1),
                            Ws2=None if lay.Ws2 is None else bf(lay.Ws2), lam=cfg.lam,
                            W3=None if lay.W3 is None else rows(lay.W3),
                            Ws3=None if lay.Ws3 is None else rows(lay.Ws3))
    return W, bf(lay.x)


def memory_bound_stages(cfg, stages, pk):
    """Achieved HBM bandwidth of the memory-bound stages from their algorithmic bytes
    and their CUDA-event times: the expert-major order (idx and gates read, perm, inv,
    row token and row gate written; the band-ordered item table, when present, is
    metadata and not counted) and the bf16 finalize (fp32 accumulator read, y written)."""
    T, d, k = cfg.T, cfg.d, cfg.k
    out = {}
    for stage, kern, nbytes in (
            ("permute", "perm_fused_kernel (+ item_order_kernel when band-ordered)", 24.0 * T * k),
            ("finalize", "f32_to_bf16_kernel", 6.0 * T * d)):
        us = stages[stage] * 1e3
        gbs = nbytes / (us * 1e-6) / 1e9 if us > 0 else None
        out[stage] = {"kernel": kern, "bytes": nbytes, "us": us, "GB/s": gbs,
                      "frac": None if gbs is None else gbs / pk["hbm_gbs"]}
    return out


def measure_config(cfg, args, world, local, with_clocks):
    """Times one workload: device-resident layer forwards (value), per-stage event
    times, and end to end with host copies.  Returns the numbers and the layer."""
    import torch
    import torch.distributed as dist

    from paper_2608_17402_gb300 import moevie

    lay = workloads.make_layer(cfg)
    W, x = _device_layer(cfg, lay, moevie, torch)
    y = torch.empty((cfg.T, cfg.d), dtype=torch.bfloat16, device="cuda")
    ws = moevie.Workspace(cfg.T, cfg.d, cfg.E, cfg.k, cfg.h, cfg.h_s)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device="cuda")
    stream = torch.cuda.current_stream()

    # routing by-products once (touched experts for the byte count)
    _, rt = moevie.moevie_moe_forward(W, x, ws, y=y, routing=True)
    counts = rt["counts"].cpu().numpy()
    code, detail = moevie.moevie_get_device_status(ws)
    if code != 0:
        raise RuntimeError(f"device status {code} {detail}")
    work = layer_work(cfg, counts, moevie.moevie_shared_groups(cfg.T, cfg.d, cfg.E, cfg.k, cfg.h, cfg.h_s))

    for _ in range(args.warmup):
        moevie.moevie_moe_forward(W, x, ws, y=y)
    torch.cuda.synchronize()

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()

    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    clk = ClockSampler(local) if with_clocks else None
    if clk is not None:
        clk.__enter__()
    try:
        barrier()
        n0 = moevie.moevie_launch_count()
        for i in range(args.steps):
            flush.zero_()                      # L2 flush outside the timed window
            starts[i].record(stream)
            moevie.moevie_moe_forward(W, x, ws, y=y)
            ends[i].record(stream)
        barrier()
        launches = moevie.moevie_launch_count() - n0
    finally:
        if clk is not None:
            clk.__exit__(None, None, None)
    ms = statistics.mean(s.elapsed_time(e) for s, e in zip(starts, ends))

    # per-stage times (events recorded between the launches, same stream)
    nstage = len(moevie.FORWARD_STAGES)
    stage_ms = np.zeros(nstage)
    for i in range(args.steps):
        evs = [torch.cuda.Event(enable_timing=True) for _ in range(nstage + 1)]
        for e in evs:
            e.record(stream)                   # creates the CUDA event handles
        flush.zero_()
        moevie.moevie_test_moe_forward_events(W, x, ws, evs, y=y)
        torch.cuda.synchronize()
        stage_ms += np.array([evs[j].elapsed_time(evs[j + 1]) for j in range(nstage)])
    stage_ms /= args.steps
    stages = dict(zip(moevie.FORWARD_STAGES, stage_ms.tolist()))

    # end to end through the C ABI from and to host memory (pinned): moevie_moe_forward_host
    # copies token chunks in and out on its own streams, overlapped with the layer; the
    # workspace sized for T serves any chunk
    x_host = torch.from_numpy(np.ascontiguousarray(lay.x).view(np.int16)).view(torch.bfloat16).pin_memory()
    y_host = torch.empty((cfg.T, cfg.d), dtype=torch.bfloat16).pin_memory()
    chunks = moevie.host_chunks(cfg.T)
    for _ in range(2):
        moevie.moevie_moe_forward_host(W, x_host, y_host, x, y, ws, chunks)
    e2e_s = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    e2e_e = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    barrier()
    for i in range(args.steps):
        flush.zero_()
        e2e_s[i].record(stream)
        moevie.moevie_moe_forward_host(W, x_host, y_host, x, y, ws, chunks)
        e2e_e[i].record(stream)
    barrier()
    e2e_ms = statistics.mean(s.elapsed_time(e) for s, e in zip(e2e_s, e2e_e))
    code, detail = moevie.moevie_get_device_status(ws)
    if code != 0:
        raise RuntimeError(f"device status {code} {detail}")
    bwd = None
    if not args.no_backward:   # the training path
        bwd = measure_backward(cfg, W, x, rt["idx"], args, flush, stream)
    del ws, flush, W, x, y
    torch.cuda.empty_cache()
    return {"ms": ms, "e2e_ms": e2e_ms, "e2e_chunks": chunks, "stages": stages, "work": work, "launches": int(launches),
            "clocks": None if clk is None else clk.summary(), "backward": bwd}, lay


def measure_backward(cfg, W, x, idx, args, flush, stream):
    """CUDA-event time of moevie_moe_backward (inputs resident, L2 flushed between calls)
    and its GEMM rate: grouped GEMMs of 2 T k d h FLOPs each -- GELU: up-projection again,
    dy W2^T, du W1^T, dW2, dW1 (5); SwiGLU: gate and up again, dy W2^T, du W1^T, dv W3^T,
    dW2, dW1, dW3 (8) -- plus dW_r = x^T ds (2 T d E), and the shared expert's own GEMMs
    (the same 5 or 8, of 2 T d h_s FLOPs each)."""
    import torch

    from paper_2608_17402_gb300 import moevie
    T, d, E, k, h = cfg.T, cfg.d, cfg.E, cfg.k, cfg.h
    g = torch.Generator(device="cuda")
    g.manual_seed(cfg.seed + 17)
    dy = torch.randn((T, d), generator=g, device="cuda").to(torch.bfloat16)
    swiglu = cfg.act == "swiglu"
    bws = moevie.BackwardWorkspace(T, d, E, k, h, h_s=cfg.h_s, swiglu=swiglu)
    steps = max(1, min(args.steps, 10))
    for _ in range(max(1, min(args.warmup, 3))):
        moevie.moevie_moe_backward(W, x, dy, idx, bws)
    torch.cuda.synchronize()
    st = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    en = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    for i in range(steps):
        flush.zero_()
        st[i].record(stream)
        moevie.moevie_moe_backward(W, x, dy, idx, bws)
        en[i].record(stream)
    torch.cuda.synchronize()
    code, detail = moevie.moevie_get_device_status(bws)
    if code != 0:
        raise RuntimeError(f"backward device status {code} {detail}")
    ms = statistics.mean(a.elapsed_time(b) for a, b in zip(st, en))
    flops = (16.0 if swiglu else 10.0) * T * d * (k * h + cfg.h_s) + 2.0 * T * d * E
    del bws, dy
    return {"us": ms * 1e3, "flops": flops, "tflops": flops / (ms / 1e3) / 1e12, "steps": steps,
            "what": "moevie_moe_backward: dx, dW_r, dW1, dW2 (dW3 for SwiGLU; dWs1, dWs2, dWs3 with a shared "
                    "expert) of sum(dy . y), selection held fixed"}


def summarise(cfg, m, pk, world):
    """Throughput, dominant-kernel roofline and layer roofline of one measured workload."""
    stages, work, ms = m["stages"], m["work"], m["ms"]
    dom = max(("up_gemm", "down_gemm"), key=lambda s: stages[s])
    dom_flops = work["flops_up_gemm"] if dom == "up_gemm" else work["flops_down_gemm"]
    achieved = dom_flops / (stages[dom] / 1e3) / 1e12
    t_roof = max(work["flops"] / (pk["bf16_tflops"] * 1e12), work["bytes"] / (pk["hbm_gbs"] * 1e9))
    roof = {"bound": "tensor", "kernel": f"grouped_gemm_kernel ({dom})", "achieved": achieved,
            "peak": pk["bf16_tflops"], "unit": "TFLOP/s", "frac": achieved / pk["bf16_tflops"],
            "traffic": captured_traffic(cfg.name, dom),
            "peak_source": pk["source"] + " bf16 burst (of measured)"}
    layer = {"flops": work["flops"], "bytes": work["bytes"], "roofline_us": t_roof * 1e6,
             "frac": t_roof / (ms / 1e3), "touched_experts": work["touched_experts"]}
    return roof, layer, world * cfg.T / (ms / 1e3)


def run_ours(args, rank, world):
    import torch
    import torch.distributed as dist  # noqa: F401

    import __graft_entry__
    from paper_2608_17402_gb300.replicas import max_over_ranks

    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    __graft_entry__.build()
    cfg = workloads.CONFIGS[args.config]
    m, lay = measure_config(cfg, args, world, local, with_clocks=True)
    ms, e2e_ms = max_over_ranks([m["ms"], m["e2e_ms"]], device="cuda")   # slowest rank
    m["ms"], m["e2e_ms"] = ms, e2e_ms

    # the other layer workloads, one GPU only (device-resident numbers and stages)
    extra = {}
    if world == 1 and args.extra:
        for name in [n for n in args.extra.split(",") if n and n != cfg.name]:
            c2 = workloads.CONFIGS[name]
            mc, _ = measure_config(c2, args, 1, local, with_clocks=False)
            roof, layer, value = summarise(c2, mc, peaks(), 1)
            extra[name] = {"workload": f"{c2.name}: {c2.note}", "tokens_per_s": value,
                           "us_per_layer": mc["ms"] * 1e3, "layer_roofline_us": layer["roofline_us"],
                           "layer_frac": layer["frac"], "dominant": roof,
                           "stages_us": {k: v * 1e3 for k, v in mc["stages"].items()},
                           "memory_bound": memory_bound_stages(c2, mc["stages"], peaks()),
                           "e2e_tokens_per_s": c2.T / (mc["e2e_ms"] / 1e3)}
            if mc.get("backward"):
                extra[name]["backward"] = mc["backward"]
    if rank != 0:
        return

    pk = peaks()
    roof, layer, value = summarise(cfg, m, pk, world)
    layer["peaks"] = pk
    out = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "us_per_layer": ms * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": f"{cfg.name}: {cfg.note}", "T": cfg.T, "d": cfg.d, "E": cfg.E, "k": cfg.k,
                   "h": cfg.h, "h_s": cfg.h_s, "act": cfg.act, "lambda": cfg.lam, "seed": cfg.seed,
                   "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
                   "l2": f"flushed between steps ({L2_FLUSH_BYTES >> 20} MiB write outside the timed window)"},
        "roofline": roof,
        "layer_roofline": layer,
        "stages_ms": m["stages"],
        "memory_bound": memory_bound_stages(cfg, m["stages"], pk),
        "e2e": {"value": world * cfg.T / (e2e_ms / 1e3), "unit": "tokens/s",
                "h2d_bytes_per_step": cfg.T * cfg.d * 2, "d2h_bytes_per_step": cfg.T * cfg.d * 2,
                "api": "moevie_moe_forward_host", "token_chunks": m["e2e_chunks"]},
        "gpu_launches": m["launches"],
        "clocks": m["clocks"],
    }
    if m.get("backward"):
        out["backward"] = m["backward"]
    if extra:
        out["per_config"] = extra
    if world == 1 and not args.no_cpu_baseline:
        out["cpu_baseline"] = cpu_baseline(lay)
    print(json.dumps(out), flush=True)


CALIBRATION_SHAPES = ((16384, 4096, 8192), (8192, 8192, 8192), (65536, 1664, 3328), (65536, 1664, 512))


def gemm_calibration(args):
    """The grouped GEMM kernel on plain dense problems, beside cuBLAS on the same shapes:
    moevie_shared_expert runs it twice (T x d by d x h_s with the GELU epilogue, then
    T x h_s by h_s x d), both operands by TMA, no gather, no reductions.  This separates
    the kernel's main loop from what the grouped layer adds (partial m-tiles, the token
    gather, the y reductions).  L2 flushed before every timed call; CUDA events; median
    of `steps` calls."""
    import torch

    from paper_2608_17402_gb300 import moevie
    torch.cuda.set_device(0)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device="cuda")
    pk = peaks()

    def timeit(fn):
        for _ in range(max(3, args.warmup)):
            fn()
        torch.cuda.synchronize()
        ts = []
        for _ in range(max(1, args.steps)):
            flush.zero_()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            fn()
            b.record()
            torch.cuda.synchronize()
            ts.append(a.elapsed_time(b))
        return statistics.median(ts) * 1e3   # µs

    g = torch.Generator(device="cuda")
    g.manual_seed(0)
    for T, d, hs in CALIBRATION_SHAPES:
        x = torch.randn((T, d), generator=g, device="cuda").to(torch.bfloat16)
        W1 = (torch.randn((d, hs), generator=g, device="cuda") / d ** 0.5).to(torch.bfloat16)
        W2 = (torch.randn((hs, d), generator=g, device="cuda") / hs ** 0.5).to(torch.bfloat16)
        ws = moevie.Workspace(T, d, 1, 1, hs, hs)
        out = torch.empty((T, d), dtype=torch.bfloat16, device="cuda")
        hbuf = torch.empty((T, hs), dtype=torch.bfloat16, device="cuda")
        ours = timeit(lambda: moevie.moevie_shared_expert(x, W1, W2, ws, out=out))
        code, detail = moevie.moevie_get_device_status(ws)
        if code != 0:
            raise RuntimeError(f"device status {code} {detail}")
        up = timeit(lambda: torch.matmul(x, W1, out=hbuf))
        down = timeit(lambda: torch.matmul(hbuf, W2, out=out))
        fl = 2.0 * T * d * hs
        print(json.dumps({"gemm_calibration": {"T": T, "d": d, "h_s": hs},
                          "ours_us": ours, "ours_tflops": 2 * fl / ours / 1e6,
                          "cublas_us": up + down, "cublas_tflops": 2 * fl / (up + down) / 1e6,
                          "cublas_up_tflops": fl / up / 1e6, "cublas_down_tflops": fl / down / 1e6,
                          "peak_bf16_tflops": pk["bf16_tflops"], "ours_frac_of_cublas": (up + down) / ours}),
              flush=True)
        del x, W1, W2, ws, out, hbuf
        torch.cuda.empty_cache()


def main():
    args = parse()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if args.gemm_calibration:
        gemm_calibration(args)
        return
    if args.impl == "reference":
        run_reference(args, rank)
        return
    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
        dist.init_process_group("nccl")
    try:
        run_ours(args, rank, world)
    finally:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()


if __name__ == "__main__":
    main()
