"""Benchmark of the rotated W4A4 hot path on GB300 (one JSON line on rank 0).

A step is one pass of the whole hot path over one batch of 2048 tokens of a
LLaMA-3-8B layer (synthetic inputs):
  * R3 + KV4: spinq_rotate_quant_kv on Q/K/V of the 2048 tokens
    (32 query heads, 8 KV heads, head_dim 128);
  * act quant: spinq_rotate_quant_act on x [2048 x 4096] (gate/up input,
    R1 merged so no online rotation, asymmetric per-token int4);
  * W4A4 GEMM: spinq_w4a4_gemm, 2048 x 4096 -> 14336 (gate/up projection);
  * R4 + act quant: spinq_rotate_quant_act on h [2048 x 14336] (down_proj
    input, online H28 (x) H512, symmetric per-token int4);
  * W4A4 GEMM: spinq_w4a4_gemm, 2048 x 14336 -> 4096 (down_proj, R4 merged
    into the weights).
The weight quantization (spinq_quant_weight) is offline and runs once before
timing.  `value` counts both GEMMs' 2*M*N*K integer ops per step over the
whole step time.  Inputs rotate over 4 independent sets (4 layers' weights and
activations, ~0.7 GB, larger than the 129 MB L2), so every step reads cold
data.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

With N > 1 (torchrun, one rank per GPU) every rank runs its own replica on its
own tokens: the path shards by tokens with no collective ("replicas only").
`--impl reference` times the CPU oracle on the host cores instead.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "W4A4 rotated-linear TOPS and rotate+quant HBM GB/s (% of GB300 peak)"
M, K, N = 2048, 4096, 14336          # gate/up projection
K2, N2, HAD2 = 14336, 4096, (28, 512)   # down_proj with online R4 = H28 (x) H512
B_KV, S_KV, HQ, HKV, D = 1, 2048, 32, 8, 128
NSETS = 4
# Measured GB300 peaks (generated MEASURED_PEAKS.json; fallbacks if absent)
FALLBACK_HBM, FALLBACK_BF16 = 6800.0, 1900.0


def peaks():
    try:
        p = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
        return float(p["hbm_gbs"]), float(p["bf16_tflops"]), "measured"
    except Exception:
        return FALLBACK_HBM, FALLBACK_BF16, "fallback"


def step_bytes_rq():
    # act quant: read fp16 x, write packed codes + alpha + beta
    return M * K * 2 + M * K // 2 + 8 * M


def step_bytes_rq2():
    # R4 + act quant (symmetric): read fp16 h, write packed codes + alpha
    return M * K2 * 2 + M * K2 // 2 + 4 * M


def step_bytes_kv():
    rq, rkv = B_KV * S_KV * HQ, B_KV * S_KV * HKV
    return rq * D * 4 + 2 * rkv * (D * 2 + D // 2 + 8)


def gemm_ops():
    return 2.0 * M * N * K


def gemm2_ops():
    return 2.0 * M * N2 * K2


def step_ops():
    return gemm_ops() + gemm2_ops()


GEMM_KERNELS = {1: ("w4a4_gemm_kernel (128 x 256 tiles)", "w4a4_gemm.cu"),
                2: ("w4a4_gemm_kernel (256 x 256 tiles)", "w4a4_gemm.cu"),
                3: ("w4a4_gemm_pair_kernel (SM pairs, 256 x 256 tiles)", "w4a4_gemm_pair.cu")}


def gemm_traffic_from_profile(profile, source):
    """DRAM bytes per GEMM launch from a committed ncu summary, or None when
    the kernel source changed since the counters were taken."""
    import hashlib
    import re
    try:
        src = os.path.join(ROOT, "paper_2405_16406_gb300", "csrc", source)
        h = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
        txt = open(os.path.join(ROOT, "profiles", profile)).read()
        if re.search(r"sha256 \(first 16 hex\): ([0-9a-f]{16})", txt).group(1) != h:
            return None
        return int(re.search(r"traffic_bytes_per_launch: (\d+)", txt).group(1))
    except Exception:
        return None


def workload_config(world):
    """The workload both arms report (the same keys and values)."""
    return {
        "workload": "llama3_8b MLP hot path for 2048 tokens: gate_up 4096->14336 (act quant, R1 merged) "
                    "+ down_proj 14336->4096 (online R4 = H28 (x) H512, act quant) "
                    "+ R3/KV4 (32 q heads, 8 kv heads, head_dim 128)",
        "M": M, "gate_up": {"K": K, "N": N, "act_quant": "asymmetric per-token int4, no online rotation"},
        "down_proj": {"K": K2, "N": N2, "online_rotation": "H28 (Paley, GF(27)) (x) H512",
                      "act_quant": "symmetric per-token int4"},
        "weights": "symmetric per-channel int4 (quantized once, not timed)",
        "l2": f"{NSETS} rotating input sets (~0.7 GB) > 129 MB L2",
        "parallelism": f"replicas{world}",
    }


# --------------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while work runs."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, dev_index: int):
        self.dev = dev_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.dev), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            threading.Thread(target=self._read, daemon=True).start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 7:
                continue
            try:
                sm.append(float(parts[0]))
                mx = float(parts[1])
            except ValueError:
                continue
            for nm, v in zip(names, parts[3:7]):
                if v.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "samples": len(sm),
                "reasons": sorted(reasons)}


# --------------------------------------------------------------------------- ours
def run_ours(args, rank, world, local_rank):
    import torch

    from paper_2405_16406_gb300 import replicas, spinq

    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream()
    hbm_peak, bf16_peak, peak_kind = peaks()
    fp8_peak = 2.0 * bf16_peak  # nominal e4m3 : bf16 dense ratio on GB300 is 2

    gen = torch.Generator(device=dev)
    gen.manual_seed(replicas.input_seed(1000, rank))

    def acts(rows, cols, frac, factor):
        x = torch.randn(rows, cols, generator=gen, device=dev)
        cols_idx = torch.randperm(cols, generator=gen, device=dev)[: max(1, int(round(frac * cols)))]
        x[:, cols_idx] *= factor
        return x.half()

    def swiglu_acts(rows, cols, frac, factor):
        # down_proj input: a * SiLU(b), a few channels scaled up
        a = torch.randn(rows, cols, generator=gen, device=dev)
        b = torch.randn(rows, cols, generator=gen, device=dev)
        h = a * torch.nn.functional.silu(b)
        del a, b
        cols_idx = torch.randperm(cols, generator=gen, device=dev)[: max(1, int(round(frac * cols)))]
        h[:, cols_idx] *= factor
        return h.half()

    sets = []
    for _ in range(NSETS):
        x = acts(M, K, 0.01, 30.0)
        w = (torch.randn(N, K, generator=gen, device=dev) * 0.02).half()
        qw = spinq.quant_weight(w, None)                       # offline, not timed
        del w
        h = swiglu_acts(M, K2, 0.005, 100.0)
        w2 = (torch.randn(N2, K2, generator=gen, device=dev) * 0.02).half()
        qw2 = spinq.quant_weight(w2, HAD2)                     # R4 merged, offline, not timed
        del w2
        q = torch.randn(B_KV, S_KV, HQ, D, generator=gen, device=dev).half()
        k = torch.randn(B_KV, S_KV, HKV, D, generator=gen, device=dev).half()
        v = torch.randn(B_KV, S_KV, HKV, D, generator=gen, device=dev).half()
        sets.append((x, qw, q, k, v, h, qw2))
    qa_out = [spinq.ActCodes(torch.empty(M, K // 2, dtype=torch.uint8, device=dev),
                             torch.empty(M, dtype=torch.float32, device=dev),
                             torch.empty(M, dtype=torch.float32, device=dev)) for _ in range(NSETS)]
    qa2_out = [spinq.ActCodes(torch.empty(M, K2 // 2, dtype=torch.uint8, device=dev),
                              torch.empty(M, dtype=torch.float32, device=dev), None) for _ in range(NSETS)]
    ys = [torch.empty(M, N, dtype=torch.float16, device=dev) for _ in range(NSETS)]
    y2s = [torch.empty(M, N2, dtype=torch.float16, device=dev) for _ in range(NSETS)]
    kv_out = [None] * NSETS
    torch.cuda.synchronize()

    # eager warm-up (also fills the library's launch-configuration caches)
    def kv_fn(j):
        _, _, q, k, v = sets[j][:5]
        kv_out[j] = spinq.rotate_quant_kv(q, k, v, out=kv_out[j])

    def rq_fn(j):
        spinq.rotate_quant_act(sets[j][0], None, False, 1.0, out=qa_out[j])

    def gemm_fn(j):
        spinq.w4a4_gemm(qa_out[j], sets[j][1], y=ys[j])

    def rq2_fn(j):
        spinq.rotate_quant_act(sets[j][5], HAD2, True, 1.0, out=qa2_out[j])

    def gemm2_fn(j):
        spinq.w4a4_gemm(qa2_out[j], sets[j][6], y=y2s[j])

    fns = (kv_fn, rq_fn, gemm_fn, rq2_fn, gemm2_fn)
    names = ("kv", "rq", "gemm", "rq2", "gemm2")
    for i in range(max(args.warmup, 3)):
        for fn in fns:
            fn(i % NSETS)
    torch.cuda.synchronize()

    # Two CUDA graphs per input set, each holding the whole step (the five
    # kernels in stream order, no host launch between them):
    #  * plain: nothing else; the timed region replays these, and ms_per_step
    #    (hence `value`) comes from events around those K replays;
    #  * timed: the same kernels with timing-event nodes between them (an event
    #    node costs a few microseconds of gap, so these are kept out of the
    #    step time); a second timed loop of K replays follows the first, and
    #    the per-kernel durations (kernel_us, the rooflines) come from the
    #    event nodes of each set's last replay in it.
    # Where this PyTorch cannot put events into a graph, the second loop
    # replays one graph per (set, kernel) with events between the replays.
    def timing_event():
        try:
            return torch.cuda.Event(enable_timing=True, external=True)
        except TypeError:
            return None

    in_graph = timing_event() is not None
    plain, timed, gev = [], [], []
    for j in range(NSETS):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for fn in fns:
                fn(j)
        plain.append(g)
        if in_graph:
            evs = [timing_event() for _ in range(len(fns) + 1)]
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                evs[0].record()
                for f_i, fn in enumerate(fns):
                    fn(j)
                    evs[f_i + 1].record()
            timed.append(g)
            gev.append(evs)
        else:
            row = []
            for fn in fns:
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g):
                    fn(j)
                row.append(g)
            timed.append(row)
    torch.cuda.synchronize()
    ev = {k2: [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(args.steps)] for k2 in names}

    def step(i):
        plain[i % NSETS].replay()

    def step_timed(i):
        if in_graph:
            timed[i % NSETS].replay()
            return
        for name, g in zip(names, timed[i % NSETS]):
            ev[name][i][0].record(stream)
            g.replay()
            ev[name][i][1].record(stream)

    for i in range(max(args.warmup, 3)):
        step(i)
        step_timed(i % args.steps)
    torch.cuda.synchronize()

    # sustain ~1.5 s so the clock samples cover steady state, ending in the timed region
    sampler = ClockSampler(local_rank) if rank == 0 else None
    if sampler:
        sampler.start()
    t_end = time.time() + 1.5
    i = 0
    while time.time() < t_end:
        for _ in range(20):
            step(i)
            i += 1
        torch.cuda.synchronize()

    replicas.barrier(world)
    torch.cuda.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for s_i in range(args.steps):
        step(s_i)
    t1.record(stream)
    torch.cuda.synchronize()
    replicas.barrier(world)
    # per-kernel timed loop (same steps, with the timing nodes)
    for s_i in range(args.steps):
        step_timed(s_i)
    torch.cuda.synchronize()
    clocks = sampler.stop() if sampler else None
    ms = replicas.max_over_ranks(t0.elapsed_time(t1) / args.steps, world, device=dev)

    def avg(key):
        if in_graph:
            k_i = names.index(key)
            last = min(args.steps, NSETS)   # sets whose last replay was in the per-kernel loop
            return statistics.mean(gev[j][k_i].elapsed_time(gev[j][k_i + 1]) for j in range(last)) / 1e3
        return statistics.mean(a.elapsed_time(b) for a, b in ev[key]) / 1e3  # seconds

    t_gemm, t_rq, t_kv, t_rq2, t_gemm2 = avg("gemm"), avg("rq"), avg("kv"), avg("rq2"), avg("gemm2")
    gemm_tops = gemm_ops() / t_gemm / 1e12
    gemm2_tops = gemm2_ops() / t_gemm2 / 1e12
    kind1, kind2 = spinq.spinq_w4a4_gemm_plan(M, N, K), spinq.spinq_w4a4_gemm_plan(M, N2, K2)

    # ---- end to end through the public API with host buffers.  Every step
    # copies its inputs from pinned host memory and reads all its outputs back
    # inside the timed region.  The copies run on their own streams, pipelined
    # across steps as a serving loop would: step i + 1's inputs go up and step
    # i - 1's outputs come down while step i computes (inputs double-buffered
    # on the device, outputs rotating over the NSETS sets, host result buffers
    # double-buffered; events order every reuse).
    NB = 2
    x_h = [sets[j][0].cpu().pin_memory() for j in range(NSETS)]
    h_h = [sets[j][5].cpu().pin_memory() for j in range(NSETS)]
    qkv_h = [tuple(t.cpu().pin_memory() for t in sets[j][2:5]) for j in range(NSETS)]

    def host_out():
        return dict(y=torch.empty(M, N, dtype=torch.float16).pin_memory(),
                    y2=torch.empty(M, N2, dtype=torch.float16).pin_memory(),
                    qo=torch.empty(B_KV, S_KV, HQ, D, dtype=torch.float16).pin_memory(),
                    kc=torch.empty(B_KV, S_KV, HKV, D // 2, dtype=torch.uint8).pin_memory(),
                    vc=torch.empty(B_KV, S_KV, HKV, D // 2, dtype=torch.uint8).pin_memory(),
                    sc=[torch.empty(B_KV, S_KV, HKV, dtype=torch.float32).pin_memory() for _ in range(4)])

    outs_h = [host_out() for _ in range(NB)]
    ins_d = [dict(x=torch.empty(M, K, dtype=torch.float16, device=dev),
                  h=torch.empty(M, K2, dtype=torch.float16, device=dev),
                  q=torch.empty(B_KV, S_KV, HQ, D, dtype=torch.float16, device=dev),
                  k=torch.empty(B_KV, S_KV, HKV, D, dtype=torch.float16, device=dev),
                  v=torch.empty(B_KV, S_KV, HKV, D, dtype=torch.float16, device=dev)) for _ in range(NB)]
    s_up, s_down = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
    comp_done = {}   # step -> event on the compute stream
    up_done = {}     # step -> event on the upload stream
    down_done = {}   # step -> event on the download stream

    def upload(i):
        b, j = i % NB, i % NSETS
        if i - NB in comp_done:
            s_up.wait_event(comp_done[i - NB])       # the device input buffer is free again
        with torch.cuda.stream(s_up):
            d = ins_d[b]
            d["x"].copy_(x_h[j], non_blocking=True)
            d["h"].copy_(h_h[j], non_blocking=True)
            d["q"].copy_(qkv_h[j][0], non_blocking=True)
            d["k"].copy_(qkv_h[j][1], non_blocking=True)
            d["v"].copy_(qkv_h[j][2], non_blocking=True)
            up_done[i] = torch.cuda.Event()
            up_done[i].record(s_up)

    def compute(i):
        b, j = i % NB, i % NSETS
        stream.wait_event(up_done[i])
        if i - NSETS in down_done:
            stream.wait_event(down_done[i - NSETS])  # set j's outputs were read back
        d = ins_d[b]
        o = spinq.rotate_quant_kv(d["q"], d["k"], d["v"], out=kv_out[j])
        spinq.rotate_quant_act(d["x"], None, False, 1.0, out=qa_out[j])
        spinq.w4a4_gemm(qa_out[j], sets[j][1], y=ys[j])
        spinq.rotate_quant_act(d["h"], HAD2, True, 1.0, out=qa2_out[j])
        spinq.w4a4_gemm(qa2_out[j], sets[j][6], y=y2s[j])
        comp_done[i] = torch.cuda.Event()
        comp_done[i].record(stream)
        return o

    def download(i, o):
        j = i % NSETS
        s_down.wait_event(comp_done[i])
        if i - NB in down_done:
            s_down.wait_event(down_done[i - NB])     # (same stream: already ordered)
        with torch.cuda.stream(s_down):
            h = outs_h[i % NB]
            h["y"].copy_(ys[j], non_blocking=True)
            h["y2"].copy_(y2s[j], non_blocking=True)
            h["qo"].copy_(o.q_out, non_blocking=True)
            h["kc"].copy_(o.k_codes, non_blocking=True)
            h["vc"].copy_(o.v_codes, non_blocking=True)
            for dst, src in zip(h["sc"], (o.k_scale, o.k_zero, o.v_scale, o.v_zero)):
                dst.copy_(src, non_blocking=True)
            down_done[i] = torch.cuda.Event()
            down_done[i].record(s_down)

    def run_e2e(n):
        comp_done.clear(), up_done.clear(), down_done.clear()
        upload(0)
        for i in range(n):
            if i + 1 < n:
                upload(i + 1)
            o = compute(i)
            download(i, o)

    run_e2e(4)
    torch.cuda.synchronize()
    replicas.barrier(world)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    s_up.wait_stream(stream)
    run_e2e(args.steps)
    stream.wait_stream(s_down)
    e1.record(stream)
    torch.cuda.synchronize()
    ms_e2e = replicas.max_over_ranks(e0.elapsed_time(e1) / args.steps, world, device=dev)
    h2d = (M * K + M * K2 + B_KV * S_KV * (HQ + 2 * HKV) * D) * 2
    d2h = (M * N + M * N2) * 2 + B_KV * S_KV * HQ * D * 2 + 2 * B_KV * S_KV * HKV * D // 2 + B_KV * S_KV * HKV * 16

    # ---- isolated timing of the two memory-bound kernels: 16 back-to-back
    # launches in one graph over 16 input sets (footprint > L2), so the graph
    # launch is amortised and every launch reads cold data
    iso = {}
    if rank == 0:
        xs = [acts(M, K, 0.01, 30.0) for _ in range(16)]
        qo = [spinq.ActCodes(torch.empty(M, K // 2, dtype=torch.uint8, device=dev),
                             torch.empty(M, dtype=torch.float32, device=dev),
                             torch.empty(M, dtype=torch.float32, device=dev)) for _ in range(16)]
        hs = [sets[i % NSETS][5] if i < NSETS else swiglu_acts(M, K2, 0.005, 100.0) for i in range(8)]
        qo2 = [spinq.ActCodes(torch.empty(M, K2 // 2, dtype=torch.uint8, device=dev),
                              torch.empty(M, dtype=torch.float32, device=dev), None) for _ in range(8)]
        kvs = [(torch.randn(B_KV, S_KV, HQ, D, generator=gen, device=dev).half(),
                torch.randn(B_KV, S_KV, HKV, D, generator=gen, device=dev).half(),
                torch.randn(B_KV, S_KV, HKV, D, generator=gen, device=dev).half()) for _ in range(16)]
        kvo = [spinq.rotate_quant_kv(*t) for t in kvs]
        for name, fn in (("act_quant", lambda i: spinq.rotate_quant_act(xs[i], None, False, 1.0, out=qo[i])),
                         ("r4_quant", lambda i: spinq.rotate_quant_act(hs[i % 8], HAD2, True, 1.0, out=qo2[i % 8])),
                         ("kv_quant", lambda i: spinq.rotate_quant_kv(*kvs[i], out=kvo[i]))):
            for i in range(16):
                fn(i)
            torch.cuda.synchronize()
            gi = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gi):
                for i in range(16):
                    fn(i)
            gi.replay()
            torch.cuda.synchronize()
            e0i = torch.cuda.Event(enable_timing=True)
            e1i = torch.cuda.Event(enable_timing=True)
            e0i.record(stream)
            for _ in range(3):
                gi.replay()
            e1i.record(stream)
            torch.cuda.synchronize()
            iso[name] = e0i.elapsed_time(e1i) / 48 / 1e3
        del xs, qo, kvs, kvo, hs, qo2

    st, _ = spinq.spinq_device_status()
    if st != spinq.SPINQ_OK:
        raise RuntimeError(f"device status after bench: {spinq.spinq_status_string(st)}")

    if rank != 0:
        return None
    value = replicas.whole_job_rate(step_ops(), ms / 1e3, world) / 1e12
    rq_gbs = step_bytes_rq() / t_rq / 1e9
    rq2_gbs = step_bytes_rq2() / t_rq2 / 1e9
    kv_gbs = step_bytes_kv() / t_kv / 1e9
    out = {
        "metric": METRIC,
        "value": round(value, 2),
        "unit": "TOPS",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(ms, 5),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "int4",
        "data": "synthetic",
        "config": workload_config(world),
        "roofline": {
            "bound": "tensor", "kernel": GEMM_KERNELS[kind1][0],
            "achieved": round(gemm_tops, 1), "peak": round(fp8_peak, 1), "unit": "TFLOP/s",
            "frac": round(gemm_tops / fp8_peak, 4),
            "traffic": gemm_traffic_from_profile(f"w4a4_gemm_gate_up_M{M}_K{K}_N{N}.md", GEMM_KERNELS[kind1][1]),
            "traffic_note": "dram__bytes_read.sum + dram__bytes_write.sum per launch from the committed ncu "
                            "summary in profiles/ (not measured in this run); null when the kernel source "
                            "hash differs from the one the counters were taken with",
            "peak_note": f"e4m3 dense = 2 x {peak_kind} bf16 ({bf16_peak} TFLOP/s); "
                         "int4 codes carried as e4m3 on tcgen05 kind::f8f6f4",
        },
        "roofline_down_proj": {
            "bound": "tensor", "kernel": GEMM_KERNELS[kind2][0] + f" (down_proj {M} x {K2} -> {N2})",
            "achieved": round(gemm2_tops, 1), "peak": round(fp8_peak, 1), "unit": "TFLOP/s",
            "frac": round(gemm2_tops / fp8_peak, 4),
            "traffic": gemm_traffic_from_profile(f"w4a4_gemm_down_proj_M{M}_K{K2}_N{N2}.md", GEMM_KERNELS[kind2][1]),
        },
        "rotate_quant_roofline": {
            "bound": "hbm", "kernel": "rq_tc_kernel (R4 = H28 (x) H512 + act quant on tcgen05, 2048 x 14336, sym)",
            "achieved": round(rq2_gbs, 1), "peak": hbm_peak, "unit": "GB/s",
            "frac": round(rq2_gbs / hbm_peak, 4), "us": round(t_rq2 * 1e6, 2),
            "isolated_us": round(iso["r4_quant"] * 1e6, 2),
            "isolated_frac": round(step_bytes_rq2() / iso["r4_quant"] / 1e9 / hbm_peak, 4),
            "note": ("in-step time between the timing nodes around the kernel in the whole-step graph "
                     "(per-kernel loop)" if in_graph else "in-step time includes the graph launch")
                    + "; isolated = 16 launches per graph, cold inputs",
        },
        "act_quant_roofline": {
            "bound": "hbm", "kernel": "rq_norot_kernel (act quant, 2048 x 4096, asym)",
            "achieved": round(rq_gbs, 1), "peak": hbm_peak, "unit": "GB/s",
            "frac": round(rq_gbs / hbm_peak, 4), "us": round(t_rq * 1e6, 2),
            "isolated_us": round(iso["act_quant"] * 1e6, 2),
            "isolated_frac": round(step_bytes_rq() / iso["act_quant"] / 1e9 / hbm_peak, 4),
        },
        "kv_roofline": {
            "bound": "hbm", "kernel": "rotate_quant_kv_kernel (2048 tokens)",
            "achieved": round(kv_gbs, 1), "peak": hbm_peak, "unit": "GB/s",
            "frac": round(kv_gbs / hbm_peak, 4), "us": round(t_kv * 1e6, 2),
            "isolated_us": round(iso["kv_quant"] * 1e6, 2),
            "isolated_frac": round(step_bytes_kv() / iso["kv_quant"] / 1e9 / hbm_peak, 4),
        },
        "kernel_us": {"gemm_gate_up": round(t_gemm * 1e6, 2), "act_quant": round(t_rq * 1e6, 2),
                      "r4_act_quant": round(t_rq2 * 1e6, 2), "gemm_down_proj": round(t_gemm2 * 1e6, 2),
                      "kv_quant": round(t_kv * 1e6, 2)},
        "e2e": {"value": round(replicas.whole_job_rate(step_ops(), ms_e2e / 1e3, world) / 1e12, 2), "unit": "TOPS",
                "pipeline": "uploads, kernels and read-backs on three streams, overlapped across steps",
                "ms_per_step": round(ms_e2e, 4), "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
        "gpu_launches": len(names) * args.steps,
        "clocks": clocks,
    }
    if not args.no_configs:
        out["configs"] = run_configs(dev, hbm_peak, fp8_peak)
        st, _ = spinq.spinq_device_status()
        if st != spinq.SPINQ_OK:
            raise RuntimeError(f"device status after the config runs: {spinq.spinq_status_string(st)}")
    if not args.no_cpu_baseline:
        out["cpu_baseline"] = cpu_baseline(sample_rows=args.cpu_rows)
    return out


# --------------------------------------------------------------------------- every config at full size
def graph_us(fn, n_inputs, reps=20):
    """Mean device time of one call: `reps` calls over rotating input copies
    (more bytes than L2, so every call reads cold data) captured in one CUDA
    graph and replayed 3 times between events."""
    import torch
    for i in range(n_inputs):
        fn(i)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for i in range(reps):
            fn(i % n_inputs)
    g.replay()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(3):
        g.replay()
    e1.record()
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) * 1e3 / (3 * reps)


def _codes_check(got_packed, x_rows, had, symmetric, what):
    """Sampled rows of timed codes against the oracle: |diff| <= 1 on at most
    1e-4 of the codes (at least one allowed per row sampled, ties only)."""
    import numpy as np

    import oracle
    ref = oracle.rotate_quant_act(x_rows, had, 4, symmetric, 1.0)
    got = oracle.unpack4(np.ascontiguousarray(got_packed), symmetric)
    d = np.abs(got.astype(np.int64) - ref.codes)
    allowed = max(int(1e-4 * d.size), 8)
    if d.max(initial=0) > 1 or np.count_nonzero(d) > allowed:
        raise RuntimeError(f"{what}: timed codes differ from the oracle ({np.count_nonzero(d)} of {d.size})")
    return int(np.count_nonzero(d))


def _gemm_check(y, qa, qw, rows, what, symmetric):
    """Sampled outputs of a timed GEMM against the oracle's dequantized
    product of the same codes (fp16 output, 2e-3 relative + 1e-3 of the
    largest |y| in the sample)."""
    import numpy as np

    import oracle
    rng = np.random.default_rng(5)
    Mr = qa.codes.shape[0]
    ms = np.asarray(rows if rows is not None else rng.integers(0, Mr, 64), dtype=np.int64)
    N = qw.codes.shape[0]
    ns = rng.integers(0, N, ms.size * 8, dtype=np.int64)
    mm = np.repeat(ms, 8)
    a_codes = oracle.unpack4(qa.codes[ms].cpu().numpy(), symmetric)
    w_codes = oracle.unpack4(qw.codes.cpu().numpy(), True)
    al = qa.scale[ms].double().cpu().numpy()
    be = None if qa.zero is None else qa.zero[ms].double().cpu().numpy()
    loc = np.repeat(np.arange(ms.size), 8)
    _, yr = oracle.w4a4_linear_sampled(a_codes, al, be, w_codes, qw.scale.double().cpu().numpy(), loc, ns)
    import torch
    yg = y[torch.as_tensor(mm, device=y.device), torch.as_tensor(ns, device=y.device)].double().cpu().numpy()
    tol = 2e-3 * np.abs(yr) + 1e-3 * np.abs(yr).max()
    if not np.all(np.abs(yg - yr) <= tol):
        raise RuntimeError(f"{what}: timed GEMM outputs differ from the oracle")
    return int(ms.size * 8)


def run_configs(dev, hbm_peak, fp8_peak):
    """Every workload at its full size, each kernel timed on its own (graph of
    back-to-back calls over cold inputs), and the timed outputs of the first
    input copy checked against the oracle on sampled rows.  Inputs of copy 0
    come from synth.py (host, numpy); further copies are device clones of it
    (only there so that every call reads data that is not in L2)."""
    import numpy as np
    import torch

    from paper_2405_16406_gb300 import spinq, synth
    res = {}

    def act_out(Mr, Kr, sym):
        return spinq.ActCodes(torch.empty(Mr, Kr // 2, dtype=torch.uint8, device=dev),
                              torch.empty(Mr, dtype=torch.float32, device=dev),
                              None if sym else torch.empty(Mr, dtype=torch.float32, device=dev))

    def copies(t, n):
        return [t] + [t.clone() for _ in range(n - 1)]

    def linear(case, tag, gemm_bound):
        x0 = torch.from_numpy(case.x).to(dev)
        w0 = torch.from_numpy(case.w).to(dev)
        qw0 = spinq.quant_weight(w0, case.had)
        del w0
        Mr, Kr, Nr = case.M, case.K, case.N
        nx = max(2, min(16, int(np.ceil(2 * 129e6 / max(1, x0.numel() * 2)))))
        xs = copies(x0, nx)
        outs = [act_out(Mr, Kr, case.act_symmetric) for _ in range(nx)]
        rq_us = graph_us(lambda i: spinq.rotate_quant_act(xs[i], case.had, case.act_symmetric, case.clip,
                                                          out=outs[i]), nx)
        rq_bytes = Mr * Kr * 2 + Mr * Kr // 2 + (4 if case.act_symmetric else 8) * Mr
        w_bytes = Nr * Kr // 2
        nw = max(2, min(16, int(np.ceil(2 * 129e6 / w_bytes))))
        qws = [qw0] + [spinq.WeightCodes(qw0.codes.clone(), qw0.scale.clone(), qw0.rowsum.clone())
                       for _ in range(nw - 1)]
        ys = [torch.empty(Mr, Nr, dtype=torch.float16, device=dev) for _ in range(nw)]
        ws = spinq.gemm_workspace(Mr, Nr, Kr, dev) if Mr <= 256 else None   # calls run in stream order
        g_us = graph_us(lambda i: spinq.w4a4_gemm_splitk(outs[i % nx], qws[i], workspace=ws, y=ys[i]) if Mr <= 256
                        else spinq.w4a4_gemm(outs[i % nx], qws[i], y=ys[i]), nw)
        torch.cuda.synchronize()
        rows = np.unique(np.linspace(0, Mr - 1, min(Mr, 8)).astype(np.int64))
        flips = _codes_check(outs[0].codes[torch.as_tensor(rows, device=dev)].cpu().numpy(), case.x[rows],
                             case.had, case.act_symmetric, tag + " rotate+quant")
        # the GEMM of call i used activation copy i % nx and weight copy i: copy 0 of both
        nchk = _gemm_check(ys[0], outs[0], qw0, rows, tag + " GEMM", case.act_symmetric)
        ops = 2.0 * Mr * Nr * Kr
        rq = {"us": round(rq_us, 3), "bytes": rq_bytes, "gbs": round(rq_bytes / rq_us / 1e3, 1),
              "frac_hbm": round(rq_bytes / rq_us / 1e3 / hbm_peak, 4)}
        gm = {"us": round(g_us, 3), "tops": round(ops / g_us / 1e6, 1),
              "kernel_plan": spinq.spinq_w4a4_gemm_splitk_plan(Mr, Nr, Kr) if Mr <= 256
              else spinq.spinq_w4a4_gemm_plan(Mr, Nr, Kr)}
        if gemm_bound == "tensor":
            gm["frac_e4m3"] = round(ops / g_us / 1e6 / fp8_peak, 4)
        else:
            gbytes = w_bytes + Mr * Kr // 2 + 2 * Mr * Nr
            gm["bytes"] = gbytes
            gm["frac_hbm"] = round(gbytes / g_us / 1e3 / hbm_peak, 4)
        r = {"M": Mr, "K": Kr, "N": Nr, "had": case.had, "rotate_quant": rq, "gemm": gm,
             "checked": f"{rows.size} rows of codes ({flips} tie flips), {nchk} GEMM outputs vs oracle"}
        del xs, outs, qws, ys
        torch.cuda.empty_cache()
        return r

    res["c1_tiny_16x256x512_h256"] = linear(synth.tiny_linear(), "config 1", "latency")
    for Mr in (1, 8, 16, 128, 8192):
        bound = "tensor" if Mr >= 2048 else "hbm"
        res[f"c5_up_M{Mr}_h12xh256"] = linear(synth.llama32_3b_up(M=Mr), f"config 5 up M={Mr}", bound)
        res[f"c5_down_M{Mr}_h8192"] = linear(synth.llama32_3b_down(M=Mr), f"config 5 down M={Mr}", bound)

    # config 4 at full size: B = 8, S = 4096 (one call moves 708.8 MB > L2)
    kv = synth.kv_case()
    q, k, v = (torch.from_numpy(t).to(dev) for t in (kv.q, kv.k, kv.v))
    o = spinq.rotate_quant_kv(q, k, v)
    kv_us = graph_us(lambda i: spinq.rotate_quant_kv(q, k, v, out=o), 1, reps=6)
    torch.cuda.synchronize()
    B, S, Hq, Hkv, Dd = kv.B, kv.S, kv.Hq, kv.Hkv, kv.D
    kv_bytes = B * S * Hq * Dd * 4 + 2 * B * S * Hkv * (Dd * 2 + Dd // 2 + 8)
    import oracle
    sel = np.random.default_rng(3).integers(0, B * S, 64)
    kr = kv.k.reshape(B * S, Hkv, Dd)[sel]
    ref = oracle.rotate_quant_kv(kv.q.reshape(B * S, 1, Hq, Dd)[sel], kr[:, None], kv.v.reshape(B * S, Hkv, Dd)[sel][:, None],
                                 kv.had)
    got = oracle.unpack4(o.k_codes.reshape(B * S, Hkv, Dd // 2)[torch.as_tensor(sel, device=dev)].cpu().numpy(), False)
    d = np.abs(got.reshape(-1) - ref.k_codes.reshape(-1))
    if d.max() > 1 or np.count_nonzero(d) > max(int(1e-4 * d.size), 8):
        raise RuntimeError("config 4: timed K codes differ from the oracle")
    res["c4_kv_B8_S4096_Hq32_Hkv8_D128"] = {
        "us": round(kv_us, 2), "bytes": kv_bytes, "gbs": round(kv_bytes / kv_us / 1e3, 1),
        "frac_hbm": round(kv_bytes / kv_us / 1e3 / hbm_peak, 4),
        "checked": f"K codes of 64 sampled tokens ({np.count_nonzero(d)} tie flips) vs oracle"}
    del q, k, v, o
    torch.cuda.empty_cache()
    res.update(cayley_records(dev))
    res.update(variant8_records(dev, hbm_peak, fp8_peak))
    res.update(attention_records(dev, hbm_peak))
    res.update(fused_down_proj_records(dev, fp8_peak))
    return res


def fused_down_proj_records(dev, fp8_peak):
    """Config 3's down_proj (2048 x 14336 -> 4096, online H28 (x) H512) as one
    call (spinq_rotated_linear), plain and with random signs (R = S H), over
    4 input sets, against the same two kernels called separately."""
    import numpy as np
    import torch

    import oracle
    from paper_2405_16406_gb300 import spinq, synth
    c = synth.llama3_8b_down_proj()
    xt, wt = torch.from_numpy(c.x).to(dev), torch.from_numpy(c.w).to(dev)
    xs = [xt] + [xt.clone() for _ in range(3)]
    signs = np.random.default_rng(17).choice([-1.0, 1.0], c.K)
    mask = spinq.sign_mask(signs)
    out = {}
    ops = 2.0 * c.M * c.N * c.K
    for tag, m in (("plain", None), ("random_signs", mask)):
        qw = spinq.quant_weight(wt, c.had) if m is None else spinq.quant_weight_signed(wt, c.had, m)
        ws = [torch.empty(spinq.spinq_rotated_linear_workspace_bytes(c.M, c.K), dtype=torch.uint8, device=dev)
              for _ in range(4)]
        ys = [torch.empty(c.M, c.N, dtype=torch.float16, device=dev) for _ in range(4)]
        us = graph_us(lambda i: spinq.rotated_linear(xs[i], c.had, qw, signs=m, y=ys[i], workspace=ws[i]), 4)
        torch.cuda.synchronize()
        # timed output of set 0, 2 rows, against the oracle's product of the handed-over codes
        rows = np.array([5, 1500])
        codes = ws[0][: c.M * c.K // 2].view(c.M, c.K // 2)[torch.as_tensor(rows, device=dev)].cpu().numpy()
        alpha = ws[0][c.M * c.K // 2:].view(torch.float32)[: c.M][torch.as_tensor(rows, device=dev)]
        ga, gw = oracle.unpack4(codes, True), oracle.unpack4(qw.codes.cpu().numpy(), True)
        ref = oracle.w4a4_linear(oracle.QuantAct(ga, None, alpha.double().cpu().numpy(), None, None),
                                 oracle.QuantWeight(gw, None, qw.scale.double().cpu().numpy(), gw.sum(1), None)).y
        got = ys[0][torch.as_tensor(rows, device=dev)].double().cpu().numpy()
        if not np.allclose(got, ref, rtol=2e-3, atol=1e-3 * np.abs(ref).max()):
            raise RuntimeError(f"rotated_linear {tag}: timed output differs from the oracle")
        rec = {"us": round(us, 2), "tops": round(ops / us / 1e6, 1), "frac_e4m3": round(ops / us / 1e6 / fp8_peak, 4)}
        if m is None:
            outs = [spinq.ActCodes(torch.empty(c.M, c.K // 2, dtype=torch.uint8, device=dev),
                                   torch.empty(c.M, device=dev), None) for _ in range(4)]
            rec["rotate_quant_alone_us"] = round(graph_us(lambda i: spinq.rotate_quant_act(xs[i], c.had, True, 1.0,
                                                                                           out=outs[i]), 4), 2)
            rec["gemm_alone_us"] = round(graph_us(lambda i: spinq.w4a4_gemm(outs[i], qw, y=ys[i]), 4), 2)
        out[f"f1_rotated_linear_down_proj_{tag}"] = rec
        del qw, ws, ys
    del xs
    torch.cuda.empty_cache()
    return out


def attention_records(dev, hbm_peak):
    """Config 4's KV path with RoPE in front of R3 (B 8, S 4096, 32 q / 8 kv
    heads, D 128), and decode attention of one query per head over the 4-bit
    cache it writes; both against HBM."""
    import numpy as np
    import torch

    import oracle
    from paper_2405_16406_gb300 import spinq, synth
    kv = synth.kv_case()
    B, S, Hq, Hkv, Dd = kv.B, kv.S, kv.Hq, kv.Hkv, kv.D
    th = 500000.0 ** (-2.0 * np.arange(Dd // 2) / Dd)
    ang = np.arange(S)[:, None] * th[None, :]
    cs = torch.from_numpy(np.stack([np.cos(ang), np.sin(ang)], -1).astype(np.float32)).to(dev)
    pos = torch.arange(S, dtype=torch.int32, device=dev).repeat(B, 1)
    q, k, v = (torch.from_numpy(t).to(dev) for t in (kv.q, kv.k, kv.v))
    cache = spinq.rope_rotate_quant_kv(q, k, v, pos, cs)
    rope_us = graph_us(lambda i: spinq.rope_rotate_quant_kv(q, k, v, pos, cs, out=cache), 1, reps=6)
    rope_bytes = B * S * Hq * Dd * 4 + 2 * B * S * Hkv * (Dd * 2 + Dd // 2 + 8) + B * S * 4
    rng = np.random.default_rng(11)
    qd = torch.from_numpy((rng.standard_normal((B, Hq, Dd)) * 2).astype(np.float16)).to(dev)
    # four caches (4 x 37.9 MB, more than the 129 MB L2): each timed call reads a cold cache
    caches = [cache] + [spinq.KVCodes(None, *(t.clone() for t in (cache.k_codes, cache.k_scale, cache.k_zero,
                                                                   cache.v_codes, cache.v_scale, cache.v_zero)))
                        for _ in range(3)]
    outs = [torch.empty_like(qd) for _ in range(4)]
    ws = torch.empty(spinq.spinq_decode_attention_workspace_bytes(B, S, Hq, Hkv, Dd), dtype=torch.uint8, device=dev)
    att_us = graph_us(lambda i: spinq.decode_attention_kv4(qd, caches[i], out=outs[i], workspace=ws), 4)
    torch.cuda.synchronize()
    att_bytes = B * S * Hkv * (Dd + 16) + 2 * B * Hq * Dd * 2
    # timed output of batch 0 against the oracle on the same codes
    kc = oracle.unpack4(cache.k_codes[:1].cpu().numpy(), False)
    vc = oracle.unpack4(cache.v_codes[:1].cpu().numpy(), False)
    kd = oracle.dequant_kv(kc, cache.k_scale[:1].double().cpu().numpy(), cache.k_zero[:1].double().cpu().numpy())
    vd = oracle.dequant_kv(vc, cache.v_scale[:1].double().cpu().numpy(), cache.v_zero[:1].double().cpu().numpy())
    ref = oracle.decode_attention(qd[:1].double().cpu().numpy(), kd, vd)
    got = outs[0][:1].double().cpu().numpy()
    if not np.all(np.abs(got - ref) <= 2e-3 * np.abs(ref) + 2e-3 * np.abs(ref).max()):
        raise RuntimeError("decode attention: timed output differs from the oracle")
    del q, k, v, cache, caches
    torch.cuda.empty_cache()
    return {
        "f2_rope_r3_kv4_B8_S4096": {"us": round(rope_us, 2), "bytes": rope_bytes,
                                     "frac_hbm": round(rope_bytes / rope_us / 1e3 / hbm_peak, 4),
                                     "kernel": "rotate_quant_kv_kernel with the RoPE stage"},
        "f2_decode_attention_kv4_B8_S4096_Hq32_Hkv8_D128": {
            "us": round(att_us, 2), "bytes": att_bytes, "frac_hbm": round(att_bytes / att_us / 1e3 / hbm_peak, 4),
            "chunks": int(ws.numel() // (B * Hq * (Dd + 2) * 4)),
            "kernel": "attn_partial_kernel + attn_combine_kernel",
            "checked": "batch 0's 32 heads vs the oracle on the same codes"}}


def variant8_records(dev, hbm_peak, fp8_peak):
    """W4A8 and W-fp8-A-fp8 at the LLaMA-3-8B MLP shapes (2048 tokens):
    gate_up 4096 -> 14336 (no rotation) and down_proj 14336 -> 4096 (online
    H28 (x) H512).  Quantizers against HBM (read 2K + write the codes and
    scales), GEMMs against the e4m3 peak; W4A8 runs 2 M N K multiply-adds on
    the tensor core (two code planes) for M N K useful ones."""
    import numpy as np
    import torch

    import oracle
    from paper_2405_16406_gb300 import spinq, synth
    out = {}
    for tag, case in (("gate_up", synth.llama3_8b_gate_up()), ("down_proj", synth.llama3_8b_down_proj())):
        Mr, Kr, Nr = case.M, case.K, case.N
        xt, wt = torch.from_numpy(case.x).to(dev), torch.from_numpy(case.w).to(dev)
        nx = 4
        xs = [xt] + [xt.clone() for _ in range(nx - 1)]
        for variant, afmt, wfmt in (("w4a8", spinq.SPINQ_FMT_INT8_PLANES, spinq.SPINQ_FMT_INT4_BYTES),
                                    ("fp8", spinq.SPINQ_FMT_E4M3, spinq.SPINQ_FMT_E4M3)):
            sym = case.act_symmetric or variant == "fp8"
            outs = [spinq.rotate_quant_act8(xs[i], case.had, afmt, sym) for i in range(nx)]
            rq_us = graph_us(lambda i: spinq.rotate_quant_act8(xs[i], case.had, afmt, sym, out=outs[i]), nx)
            planes = 2 if variant == "w4a8" else 1
            rq_bytes = Mr * Kr * 2 + planes * Mr * Kr + (4 if sym else 8) * Mr
            wq = spinq.quant_weight8(wt, case.had, wfmt)
            ys = [torch.empty(Mr, Nr, dtype=torch.float16, device=dev) for _ in range(2)]
            if variant == "w4a8":
                g_us = graph_us(lambda i: spinq.w4a8_gemm(outs[i % nx], wq, y=ys[i]), 2)
            else:
                g_us = graph_us(lambda i: spinq.fp8_gemm(outs[i % nx], wq, y=ys[i]), 2)
            torch.cuda.synchronize()
            # timed output of copy 0 against the oracle on 4 rows x 256 columns
            rows = np.array([0, 700, 1400, 2047])
            cols = np.arange(0, Nr, Nr // 256)
            sel = torch.as_tensor(rows, device=dev)
            a_rows = outs[0].codes[sel].cpu().numpy()
            if variant == "w4a8":
                c = (oracle.e4m3_to_f64(a_rows[:, :Kr]) + oracle.e4m3_to_f64(a_rows[:, Kr:])).astype(np.int32)
                wc = oracle.e4m3_to_f64(wq.codes[torch.as_tensor(cols, device=dev)].cpu().numpy()).astype(np.int32)
                zero = None if sym else outs[0].zero[sel].double().cpu().numpy()
                qa = oracle.QuantAct(c if sym else c + 128, None, outs[0].scale[sel].double().cpu().numpy(), zero, None)
                qw = oracle.QuantWeight(wc, None, wq.scale[torch.as_tensor(cols, device=dev)].double().cpu().numpy(),
                                        wc.sum(1), None)
                yr = oracle.w4a8_linear(qa, qw).y
            else:
                yr = oracle.fp8_linear(a_rows, outs[0].scale[sel].double().cpu().numpy(),
                                       wq.codes[torch.as_tensor(cols, device=dev)].cpu().numpy(),
                                       wq.scale[torch.as_tensor(cols, device=dev)].double().cpu().numpy())
            yg = ys[0][sel][:, torch.as_tensor(cols, device=dev)].double().cpu().numpy()
            if not np.allclose(yg, yr, rtol=2e-3, atol=1e-3 * np.abs(yr).max()):
                raise RuntimeError(f"{variant} {tag}: timed GEMM outputs differ from the oracle")
            ops = 2.0 * Mr * Nr * Kr
            out[f"f3_{variant}_{tag}_{Mr}x{Kr}x{Nr}"] = {
                "rotate_quant": {"us": round(rq_us, 2), "bytes": rq_bytes,
                                 "frac_hbm": round(rq_bytes / rq_us / 1e3 / hbm_peak, 4),
                                 "kernel": ("rq8_rows_kernel (one CTA per row)" if case.had is None else
                                            "rq_tc_kernel (tcgen05, E4M3 epilogue)" if variant == "fp8" else
                                            "rq_paley_kernel (int8 planes epilogue)")},
                "gemm": {"us": round(g_us, 2), "tops": round(ops / g_us / 1e6, 1),
                         "tensor_frac_e4m3": round(planes * ops / g_us / 1e6 / fp8_peak, 4),
                         "kernel": "fp8_gemm_kernel" + (" (two activation planes, K' = 2K)" if planes == 2 else "")},
                "checked": "4 rows x 256 columns of the timed output vs the oracle's product of the same codes"}
            del outs, ys, wq
            torch.cuda.empty_cache()
        del xs, xt, wt
    return out


def cayley_records(dev):
    """Cayley SGD step (Sec. 3.2) on batches of head_dim x head_dim rotations:
    32 (one R2 per layer of a 32-layer model) and 152 (one per SM).  Bound by
    fp32 FMA issue: (4 + iters) n x n products, 2 n^3 flops each, against
    the fp32 peak 152 SMs x 128 FMA/clk x 2 flops x 2.07 GHz = 80.5 TFLOP/s."""
    import numpy as np
    import torch

    import oracle
    from paper_2405_16406_gb300 import spinq
    out = {}
    n, iters = 128, 2
    peak = 152 * 128 * 2 * 2.07e9 / 1e12
    for batch in (32, 152):
        rng = np.random.default_rng(batch)
        R = np.stack([np.linalg.qr(rng.standard_normal((n, n)))[0] for _ in range(batch)]).astype(np.float32)
        g = (0.5 * rng.standard_normal((batch, n, n))).astype(np.float32)
        alpha = 0.01
        Rt, gt = torch.from_numpy(R).to(dev), torch.from_numpy(g).to(dev)
        outs = [torch.empty_like(Rt) for _ in range(2)]
        us = graph_us(lambda i: spinq.cayley_step(Rt, gt, alpha, iters, out=outs[i]), 2)
        torch.cuda.synchronize()
        ref, _ = oracle.cayley_step(R[:2].astype(np.float64), g[:2].astype(np.float64), alpha, iters)
        err = float(np.abs(outs[0][:2].cpu().numpy() - ref).max())
        if err > 5e-5:
            raise RuntimeError(f"Cayley step: timed output differs from the oracle by {err}")
        flops = batch * (4 + iters) * 2.0 * n ** 3
        tf = flops / us / 1e6
        out[f"f4_cayley_step_{batch}x{n}x{n}_iters{iters}"] = {
            "us": round(us, 2), "tflops": round(tf, 2), "bound": "alu (fp32 FMA)",
            "peak_tflops": round(peak, 1), "frac": round(tf / peak, 4),
            "frac_of_used_sms": round(tf / (peak * min(batch, 152) / 152), 4),
            "checked": f"2 rotations vs oracle, max abs diff {err:.1e}"}
    return out


# --------------------------------------------------------------------------- oracle on host cores
_ORACLE_WEIGHTS = {}


def _oracle_weights():
    """The two layers' weights quantized by the oracle: offline work, done
    once per process and never timed."""
    if not _ORACLE_WEIGHTS:
        import numpy as np

        import oracle
        from paper_2405_16406_gb300 import synth
        rng = np.random.default_rng(1)
        _ORACLE_WEIGHTS["gate_up"] = oracle.quant_weight(synth.weights(rng, N, K), None)
        _ORACLE_WEIGHTS["down_proj"] = oracle.quant_weight(synth.weights(rng, N2, K2), HAD2)
    return _ORACLE_WEIGHTS["gate_up"], _ORACLE_WEIGHTS["down_proj"]


def cpu_baseline(sample_rows=1024, threads=0):
    """Time the oracle (as it stands) on a bounded sample of the same workload:
    `sample_rows` tokens through act quant + GEMM (+ their KV rows)."""
    import numpy as np

    import oracle
    from paper_2405_16406_gb300 import synth
    cores = oracle.set_threads(threads)
    qw, qw2 = _oracle_weights()
    rng = np.random.default_rng(0)
    x = synth.activations(rng, sample_rows, K, outlier_frac=0.01, factor=30.0)
    h = synth.activations(rng, sample_rows, K2, outlier_frac=0.005, factor=100.0, swiglu=True)
    kv = synth.kv_case(seed=1, B=1, S=sample_rows, Hq=HQ, Hkv=HKV, D=D)
    t0 = time.perf_counter()
    oracle.rotate_quant_kv(kv.q, kv.k, kv.v, kv.had)
    qa = oracle.rotate_quant_act(x, None, 4, False, 1.0)
    oracle.w4a4_linear(qa, qw)
    qa2 = oracle.rotate_quant_act(h, HAD2, 4, True, 1.0)
    oracle.w4a4_linear(qa2, qw2)
    dt = time.perf_counter() - t0
    ops = 2.0 * sample_rows * (N * K + N2 * K2)
    return {"value": round(ops / dt / 1e12, 6), "unit": "TOPS", "cores": cores, "kind": "oracle",
            "sample": f"{sample_rows} of {M} tokens (KV rows for the same tokens, act quant + GEMM "
                      f"{sample_rows}x{K}->{N}, R4 + act quant + GEMM {sample_rows}x{K2}->{N2}); {dt:.2f} s"}


def run_reference(args, rank, world):
    """The CPU oracle as it stands, on the host cores: every step runs the
    whole path (KV rows, act quant + gate_up GEMM, R4 + act quant + down_proj
    GEMM) on a bounded sample of `--ref-rows` tokens of the workload, and the
    line reports that measured time.  The rate (TOPS) is the sample's ops
    over the sample's time; nothing is projected to the full batch."""
    if rank != 0:
        return None
    rows = args.ref_rows
    _oracle_weights()                       # offline weight quantization, not timed
    for _ in range(args.warmup):
        cpu_baseline(sample_rows=max(1, rows // 4))
    t0 = time.perf_counter()
    vals = [cpu_baseline(sample_rows=rows) for _ in range(args.steps)]
    wall = time.perf_counter() - t0
    ms_per_step = wall / args.steps * 1e3
    ops = 2.0 * rows * (N * K + N2 * K2) * args.steps
    v = ops / wall / 1e12
    cb = dict(vals[-1])
    cb["value"] = round(v, 6)
    cb["sample"] = (f"{rows} of the workload's {M} tokens per step through every step of the path "
                    f"(KV rows for the same tokens, act quant + GEMM {rows}x{K}->{N}, R4 + act quant + GEMM "
                    f"{rows}x{K2}->{N2}); {args.steps} steps in {wall:.2f} s")
    return {
        "metric": METRIC, "value": round(v, 6), "unit": "TOPS", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_per_step, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "impl": "reference",
        "config": workload_config(world),
        "sample_tokens_per_step": rows,
        "cpu_baseline": cb,
        "e2e": {"value": round(v, 6), "unit": "TOPS", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def launch_check(args, rank, world):
    """Start-up check of the multi-rank launch (no kernels): every rank joins
    the process group (NCCL on GPUs, gloo on CPU) and rank 0 reports how many
    ranks it saw."""
    import torch
    import torch.distributed as dist
    if world > 1:
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        dev = "cpu"
        if backend == "nccl":
            torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
            dev = "cuda"
        dist.init_process_group(backend)
        t = torch.ones(1, device=dev)
        dist.all_reduce(t)
        seen = int(t.item())
        dist.destroy_process_group()
    else:
        seen = 1
    return {"launch_check": True, "n_gpus": args.gpus, "world": world, "ranks_seen": seen} if rank == 0 else None


def relaunch(args_n):
    """`--gpus N` without a launcher: run this script under
    torch.distributed.run with N ranks on this node and return its status."""
    import socket
    with socket.socket() as so:
        so.bind(("127.0.0.1", 0))
        port = so.getsockname()[1]
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", f"--nproc-per-node={args_n}",
           "--master-addr", "127.0.0.1", "--master-port", str(port), os.path.abspath(__file__)] + sys.argv[1:]
    return subprocess.call(cmd)


PROFILE_CASES = ("attention", "rope_kv", "fp8_gemm", "w4a8_gemm", "rq8_paley", "cayley", "paley", "gemm",
                 "gemm_gate_up", "decode_gemm", "decode_gemm16", "rq_h8192", "kv2048", "act_quant")


def profile_case(name, reps):
    """One kernel family on its bench workload, `reps` launches, for a
    profiler (`ncu -k ... python bench.py --profile-case NAME`): no timing,
    prints the device status.  attention: decode attention over the
    B 8, S 4096, 32/8-head, D 128 cache; rope_kv: RoPE + R3 + KV4 on B 2 of
    that cache; fp8_gemm / w4a8_gemm: the gate_up projection 2048 x 4096 ->
    14336 with E4M3 codes / 4-bit weights and 8-bit activation planes;
    rq8_paley: the 8-bit quantizer with H28 x H512 on 2048 x 14336; cayley:
    152 rotations of 128 x 128, 2 iterations; paley: the 4-bit R4 kernel on
    2048 x 14336; gemm: the W4A4 down_proj 2048 x 14336 -> 4096; gemm_gate_up:
    the W4A4 gate_up 2048 x 4096 -> 14336 (asymmetric activations);
    decode_gemm: 8 tokens through 4096 -> 14336 on the automatic route;
    decode_gemm16: 16 tokens through 3072 -> 8192 on the automatic route;
    rq_h8192: the 4-bit R4 kernel with H8192 on 8192 x 8192 (asymmetric);
    kv2048: R3 + KV4 on the step's 2048 tokens (32 / 8 heads, D 128);
    act_quant: the step's gate_up activation quantizer (2048 x 4096, no
    rotation, asymmetric)."""
    import numpy as np
    import torch

    from paper_2405_16406_gb300 import spinq, synth
    dev = torch.device("cuda", 0)
    if name == "attention":
        kv = synth.kv_case()
        cache = spinq.rotate_quant_kv(torch.from_numpy(kv.q).to(dev), torch.from_numpy(kv.k).to(dev),
                                      torch.from_numpy(kv.v).to(dev))
        qd = (torch.randn(kv.B, kv.Hq, kv.D, device=dev) * 2).half()
        fn = lambda: spinq.decode_attention_kv4(qd, cache)
    elif name == "rope_kv":
        kv = synth.kv_case(B=2)
        th = 500000.0 ** (-2.0 * np.arange(kv.D // 2) / kv.D)
        ang = np.arange(kv.S)[:, None] * th[None, :]
        cs = torch.from_numpy(np.stack([np.cos(ang), np.sin(ang)], -1).astype(np.float32)).to(dev)
        pos = torch.arange(kv.S, dtype=torch.int32, device=dev).repeat(kv.B, 1)
        q, k, v = (torch.from_numpy(t).to(dev) for t in (kv.q, kv.k, kv.v))
        fn = lambda: spinq.rope_rotate_quant_kv(q, k, v, pos, cs)
    elif name in ("fp8_gemm", "w4a8_gemm"):
        c = synth.llama3_8b_gate_up()
        x, w = torch.from_numpy(c.x).to(dev), torch.from_numpy(c.w).to(dev)
        if name == "fp8_gemm":
            qa = spinq.rotate_quant_act8(x, None, spinq.SPINQ_FMT_E4M3, True)
            qw = spinq.quant_weight8(w, None, spinq.SPINQ_FMT_E4M3)
            fn = lambda: spinq.fp8_gemm(qa, qw)
        else:
            qa = spinq.rotate_quant_act8(x, None, spinq.SPINQ_FMT_INT8_PLANES, False)
            qw = spinq.quant_weight8(w, None, spinq.SPINQ_FMT_INT4_BYTES)
            fn = lambda: spinq.w4a8_gemm(qa, qw)
    elif name in ("rq8_paley", "paley", "gemm"):
        c = synth.llama3_8b_down_proj()
        x = torch.from_numpy(c.x).to(dev)
        if name == "rq8_paley":
            fn = lambda: spinq.rotate_quant_act8(x, c.had, spinq.SPINQ_FMT_E4M3, True)
        elif name == "paley":
            fn = lambda: spinq.rotate_quant_act(x, c.had)
        else:
            qa = spinq.rotate_quant_act(x, c.had)
            qw = spinq.quant_weight(torch.from_numpy(c.w).to(dev), c.had)
            fn = lambda: spinq.w4a4_gemm(qa, qw)
    elif name == "rq_h8192":
        c = synth.llama32_3b_down(M=8192)
        x8 = torch.from_numpy(c.x).to(dev)
        fn = lambda: spinq.rotate_quant_act(x8, c.had, c.act_symmetric)
    elif name == "gemm_gate_up":
        c = synth.llama3_8b_gate_up()
        qa = spinq.rotate_quant_act(torch.from_numpy(c.x).to(dev), None, False)
        qw = spinq.quant_weight(torch.from_numpy(c.w).to(dev), None)
        fn = lambda: spinq.w4a4_gemm(qa, qw)
    elif name == "decode_gemm":
        c = synth.llama3_8b_gate_up(M=8)
        qa = spinq.rotate_quant_act(torch.from_numpy(c.x).to(dev), None, False)
        qw = spinq.quant_weight(torch.from_numpy(c.w).to(dev), None)
        fn = lambda: spinq.w4a4_gemm_splitk(qa, qw)
    elif name == "decode_gemm16":
        c = synth.llama32_3b_up(M=16)
        qa = spinq.rotate_quant_act(torch.from_numpy(c.x).to(dev), c.had, c.act_symmetric)
        qw = spinq.quant_weight(torch.from_numpy(c.w).to(dev), c.had)
        fn = lambda: spinq.w4a4_gemm_splitk(qa, qw)
    elif name == "kv2048":
        kv = synth.kv_case(B=1, S=2048)
        q, k, v = (torch.from_numpy(t).to(dev) for t in (kv.q, kv.k, kv.v))
        fn = lambda: spinq.rotate_quant_kv(q, k, v)
    elif name == "act_quant":
        c = synth.llama3_8b_gate_up()
        x = torch.from_numpy(c.x).to(dev)
        fn = lambda: spinq.rotate_quant_act(x, None, False)
    elif name == "cayley":
        rng = np.random.default_rng(0)
        R = np.stack([np.linalg.qr(rng.standard_normal((128, 128)))[0] for _ in range(152)]).astype(np.float32)
        Rt = torch.from_numpy(R).to(dev)
        G = torch.from_numpy((rng.standard_normal((152, 128, 128)) * 0.5).astype(np.float32)).to(dev)
        fn = lambda: spinq.cayley_step(Rt, G, 0.01, 2)
    else:
        raise ValueError(f"unknown profile case {name}")
    for _ in range(reps):
        fn()
    torch.cuda.synchronize()
    st = spinq.spinq_device_status()
    print(json.dumps({"profile_case": name, "reps": reps, "device_status": list(st)}))
    return 0 if st[0] == spinq.SPINQ_OK else 1


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--cpu-rows", type=int, default=1024)
    ap.add_argument("--ref-rows", type=int, default=64, help="tokens per --impl reference step")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-configs", action="store_true", help="skip the per-config full-size runs")
    ap.add_argument("--launch-check", action="store_true",
                    help="only start the ranks, join the process group and report them (no kernels)")
    ap.add_argument("--profile-case", choices=PROFILE_CASES,
                    help="run one kernel family on its bench workload --reps times and exit (for a profiler)")
    ap.add_argument("--reps", type=int, default=3, help="launches of --profile-case")
    args = ap.parse_args()

    if args.profile_case:
        sys.exit(profile_case(args.profile_case, args.reps))
    if args.gpus < 1:
        ap.error("--gpus must be at least 1")
    if "WORLD_SIZE" not in os.environ and args.gpus > 1:
        sys.exit(relaunch(args.gpus))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if world != args.gpus:
        print(f"bench.py: --gpus {args.gpus} but the launcher started {world} ranks", file=sys.stderr)
        sys.exit(2)

    if args.launch_check:
        out = launch_check(args, rank, world)
    elif args.impl == "reference":
        out = run_reference(args, rank, world)
    else:
        import torch
        import torch.distributed as dist
        if world > 1:
            torch.cuda.set_device(local_rank)
            dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
        out = run_ours(args, rank, world, local_rank)
        if world > 1:
            dist.destroy_process_group()
    if out is not None:
        print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
