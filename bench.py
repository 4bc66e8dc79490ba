"""Throughput of the NAMOH routed-attention path on GB300, one JSON line on stdout.

Step (the whole hot path over one batch): route + dispatch, RoPE at rank / cache pack,
length-aware plan, routed causal attention with the gate-weighted combine, on the
balanced prefill workload (4 sequences x 4096 tokens, H = 16, K = 4, d = 128, bf16,
RoPE base 1e4), inputs resident in HBM.  L2 (129 MB) is flushed by writing a 2 GB
buffer before every timed step, because that workload's inputs (51 MB) fit in L2.  The
flush also keeps the GPU busy while the host enqueues the step, so device time excludes
host launch gaps (checked and reported).  The headline times whole steps (events only at
the step boundaries), so the RoPE and attention kernels overlap the tail of the kernel
before them (programmatic dependent launch); a second pass with events between the
stages gives the stage breakdown and the attention kernel's duration for the roofline.

The end-to-end figure ("e2e") goes through namoh_route + namoh_prefill from pinned host
buffers: every step copies its own inputs in and its own y out, with consecutive steps
overlapped on three streams, as a server would run them.

The other prefill workloads (PR1, the skewed 32k-token workload, the H sweep at 16k tokens and
its GQA variant) are measured in the same run under "configs", each with its attention kernel's
roofline fraction and the oracle timed on the host cores beside it.  The decode workload (64
sequences with 131072-token routed prefixes, H = 32, K = 4, d = 128, 17.4 GB KV cache, 256 steps)
is reported under "decode", with the oracle timed on two of its sequences for every step.

--impl reference runs the fp64 CPU oracle (the reference arm for this path) on a
bounded sample of the same workload.  Under torchrun each rank runs its own replica
(replicas only, no collective); rank 0 prints the line.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import platform
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import namoh_inputs as ni  # noqa: E402
from paper_2609_38832_gb300 import accounting as acc  # noqa: E402

METRIC = "prefill routed-attn TFLOP/s (% bf16 peak); decode tokens/s and HBM GB/s (% peak)"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
NOMINAL_HBM_GBS = 8000.0
ATTN_SOURCES = ["paper_2609_38832_gb300/csrc/prefill_attn.cu", "paper_2609_38832_gb300/csrc/common.cuh"]
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "attn_fwd_balanced_traffic.json")


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d, "measured"
    return FALLBACK_PEAKS, "fallback"


def source_hash(files):
    h = hashlib.sha256()
    for f in files:
        h.update(open(os.path.join(ROOT, f), "rb").read())
    return h.hexdigest()[:16]


def ncu_traffic():
    """DRAM bytes per attention launch from the committed ncu summary, if it matches this source."""
    if not os.path.exists(TRAFFIC_FILE):
        return None
    d = json.load(open(TRAFFIC_FILE))
    if d.get("source_hash") != source_hash(ATTN_SOURCES):
        return None
    return d.get("dram_bytes_per_launch")


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 200 ms while running."""
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except OSError:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for name, val in zip(names, parts[4:8]):
                if val.lower() == "active":
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": float(max(mx)), "reasons": sorted(reasons),
                "samples": len(sm)}


def cpu_model():
    try:
        for line in open("/proc/cpuinfo"):
            if line.lower().startswith(("model name", "cpu part")):
                return line.split(":", 1)[1].strip()
    except OSError:
        pass
    return platform.processor() or platform.machine()


def stats(ms):
    """Summary of per-launch (or per-step) times in ms: mean, median, p10, p90."""
    a = np.asarray(ms, dtype=np.float64)
    return {"mean": float(a.mean()), "median": float(np.median(a)), "p10": float(np.percentile(a, 10)),
            "p90": float(np.percentile(a, 90)), "n": int(a.size)}


# --------------------------------------------------------------------------- oracle (CPU baseline)
def oracle_prefill_sample(wl: ni.PrefillWorkload, min_seconds: float = 10.0, max_reps: int = 64):
    """The oracle, as it stands, on the full workload (route + prefill), repeated until min_seconds."""
    import oracle
    oracle.build()
    scores = wl.scores()
    q, k, v = wl.qkv()
    threads = oracle.default_threads()
    reps, t_total = 0, 0.0
    while reps < max_reps and (reps == 0 or t_total < min_seconds):
        t0 = time.perf_counter()
        r = oracle.route(scores, wl.Kr)
        oracle.prefill(q, k, v, r["seg_offsets"], r["row_src"], r["gate"], wl.d, wl.g, wl.base, nthreads=threads)
        t_total += time.perf_counter() - t0
        reps += 1
        n = r["n"]
    flops = acc.attention_flops(n, wl.d, wl.g)
    return {"value": flops * reps / t_total / 1e12, "unit": "TFLOP/s", "cores": threads, "kind": "oracle",
            "sample": f"full {wl.name} workload (route + prefill), {reps} repetition(s), {t_total:.1f} s, "
                      f"fp64 C on {threads} host threads ({cpu_model()})",
            "seconds_per_step": t_total / reps}


# --------------------------------------------------------------------------- GPU measurement
def run_gpu(args, rank: int, world: int):
    import torch

    import paper_2609_38832_gb300 as namoh

    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", 0)))
    torch.cuda.set_device(dev)
    wl = ni.BALANCED
    pk, pk_kind = peaks()

    # ---- inputs resident in HBM
    scores_h = wl.scores()
    q_h, k_h, v_h = wl.qkv()

    def to_dev(bits):
        return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(dev)

    scores = torch.from_numpy(scores_h).to(dev)
    q, k, v = to_dev(q_h), to_dev(k_h), to_dev(v_h)
    B, T, H, K, d, g = wl.B, wl.T, wl.H, wl.K, wl.d, wl.g
    ws = namoh.Workspace()
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    ro = namoh.namoh_route(scores, wl.Kr, workspace=ws, status=status)
    q_rot = torch.empty_like(q)
    k_cache = torch.empty_like(k)
    plan = namoh.namoh_attention_plan(ro.seg_offsets, B=B, T=T, H=H, K=K, group=g)
    y = torch.empty((B, T, K, d), dtype=torch.bfloat16, device=dev)
    flush = torch.empty(2 << 30, dtype=torch.uint8, device=dev)

    def step(ev=None):
        if ev is not None:
            ev[0].record()
        namoh.namoh_route(scores, wl.Kr, workspace=ws, status=status, out=ro)
        if ev is not None:
            ev[1].record()
        namoh.namoh_rope_pack(q, k, v, ro.seg_offsets, B=B, T=T, H=H, K=K, group=g, rope_base=wl.base, q_rot=q_rot,
                              k_cache=k_cache, v_cache=v, status=status, plan=plan)
        if ev is not None:
            ev[2].record()
        namoh.namoh_attention(q_rot, k_cache, v, ro.seg_offsets, ro.row_src, ro.gate, plan, B=B, T=T, H=H, K=K,
                              group=g, y=y, status=status)
        if ev is not None:
            ev[3].record()

    clocks = ClockSampler(dev.index).__enter__()
    for _ in range(args.warmup):
        flush.fill_(1)
        step()
    torch.cuda.synchronize()
    n_seg = acc.segment_lengths(ro.seg_offsets.cpu().numpy())
    flops = acc.attention_flops(n_seg, d, g)
    # Timed region (headline): whole steps, events only at the step boundaries, so that the
    # RoPE and attention kernels can start during the kernel before them (programmatic
    # dependent launch).  A second pass with an event between every stage gives the stage
    # breakdown and the attention kernel's own duration for the roofline.
    step_ev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]
    fl_ev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]
    enqueue_s = []
    barrier(world)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for i in range(args.steps):
        fl_ev[i][0].record()
        flush.fill_(i & 0xFF)
        fl_ev[i][1].record()
        te = time.perf_counter()
        step_ev[i][0].record()
        step()
        step_ev[i][1].record()
        enqueue_s.append(time.perf_counter() - te)
    torch.cuda.synchronize()
    wall = time.perf_counter() - t0
    barrier(world)
    flush_ms = [a.elapsed_time(b) for a, b in fl_ev]
    # the host finished enqueueing each step before the flush ahead of it ended
    gapless = all(e * 1e3 < f for e, f in zip(enqueue_s, flush_ms))
    step_times = [a.elapsed_time(b) for a, b in step_ev]
    step_ms = max_over_ranks(float(np.median(step_times)), world)

    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(args.steps)]
    for i in range(args.steps):
        flush.fill_(i & 0xFF)
        step(evs[i])
    torch.cuda.synchronize()
    stage = np.array([[evs[i][j].elapsed_time(evs[i][j + 1]) for j in range(3)] for i in range(args.steps)])
    attn_ms = float(stage[:, 2].mean())  # the roofline divides by the kernel's average launch duration
    st = int(status.item())

    # ---- the RoPE/plan launch alone in each RoPE variant (Sec. 3.2: rank or global position;
    # half-split or interleaved pairs), L2 flushed before every launch.  Algorithmic bytes:
    # Q and K read, Q~ and K~ written (V serves as its own cache here), plus row_src for global.
    R = B * T * wl.Kr
    rope_bytes = 2 * (R * g * d * 2 + R * d * 2)
    rope_variants = {}
    for name, il, gp in (("half_split_rank", False, False), ("interleaved_rank", True, False),
                         ("half_split_global", False, True), ("interleaved_global", True, True)):
        evr = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]
        for i in range(args.warmup + args.steps):
            flush.fill_(i & 0xFF)
            if i >= args.warmup:
                evr[i - args.warmup][0].record()
            namoh.namoh_rope_pack(q, k, v, ro.seg_offsets, B=B, T=T, H=H, K=K, group=g, rope_base=wl.base,
                                  interleaved=il, row_src=ro.row_src if gp else None, q_rot=q_rot, k_cache=k_cache,
                                  v_cache=v, status=status, plan=plan)
            if i >= args.warmup:
                evr[i - args.warmup][1].record()
        torch.cuda.synchronize()
        ms = float(np.mean([a.elapsed_time(b) for a, b in evr]))
        nbytes = rope_bytes + (R * 4 if gp else 0)
        rope_variants[name] = {"ms": ms, "hbm_gbs": nbytes / (ms * 1e-3) / 1e9,
                               "hbm_frac": nbytes / (ms * 1e-3) / 1e9 / pk["hbm_gbs"]}
    rope_variants["bytes"] = "2 (R g d + R d) bf16 (+ 4 R for row_src under global positions), R = B T Kr"
    st |= int(status.item())

    # ---- end to end through the public API with host buffers (pinned), copies timed.
    # Every step copies its own inputs host -> device, runs namoh_route + namoh_prefill and
    # reads its own y back.  Consecutive steps overlap as in serving: the input copies of step
    # i+1 run on their own stream while step i computes and step i-1's output is read back.
    # Inputs and outputs rotate over NSET device buffer sets (NSET x 51 MB > L2), so no step
    # finds another step's inputs in L2; a set is rewritten only after the step that used it
    # has finished with it (events across the three streams).
    pin = lambda a: torch.from_numpy(np.ascontiguousarray(a)).pin_memory()  # noqa: E731
    scores_p = pin(scores_h)
    q_p, k_p, v_p = pin(q_h.view(np.int16)), pin(k_h.view(np.int16)), pin(v_h.view(np.int16))
    NSET = 4
    y_p = [torch.empty((B, T, K, d), dtype=torch.int16).pin_memory() for _ in range(NSET)]
    sets = [(torch.empty_like(scores), torch.empty(q.shape, dtype=torch.int16, device=dev),
             torch.empty(k.shape, dtype=torch.int16, device=dev), torch.empty(v.shape, dtype=torch.int16, device=dev),
             torch.empty((B, T, K, d), dtype=torch.bfloat16, device=dev)) for _ in range(NSET)]
    s_in, s_cmp, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev), torch.cuda.Stream(dev)

    def e2e_compute(j, stream=None):
        s_d, q_d, k_d, v_d, y_d = sets[j]
        r = namoh.namoh_route(s_d, wl.Kr, workspace=ws, status=status, out=ro, stream=stream)
        namoh.namoh_prefill(q_d.view(torch.bfloat16), k_d.view(torch.bfloat16), v_d.view(torch.bfloat16),
                            r.seg_offsets, r.row_src, r.gate, B=B, T=T, H=H, K=K, group=g, rope_base=wl.base,
                            y=y_d, k_cache=k_cache, workspace=ws, status=status, stream=stream)

    # one serial step first, on the current stream: sizes the shared workspace once
    for j in range(NSET):
        for dst, src in zip(sets[j][:4], (scores_p, q_p, k_p, v_p)):
            dst.copy_(src, non_blocking=True)
    e2e_compute(0)
    torch.cuda.synchronize()

    def e2e_pipeline(n):
        """n pipelined steps; returns (start event on the input stream, end event on the output stream)."""
        ev_in = [torch.cuda.Event() for _ in range(n)]
        ev_cmp = [torch.cuda.Event() for _ in range(n)]
        ev_out = [torch.cuda.Event() for _ in range(n)]
        start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        start.record(s_in)
        for i in range(n):
            j = i % NSET
            s_d, q_d, k_d, v_d, y_d = sets[j]
            with torch.cuda.stream(s_in):
                if i >= NSET:
                    s_in.wait_event(ev_cmp[i - NSET])  # step i-NSET has finished reading this set
                for dst, src in zip((s_d, q_d, k_d, v_d), (scores_p, q_p, k_p, v_p)):
                    dst.copy_(src, non_blocking=True)
                ev_in[i].record(s_in)
            with torch.cuda.stream(s_cmp):
                s_cmp.wait_event(ev_in[i])
                if i >= NSET:
                    s_cmp.wait_event(ev_out[i - NSET])  # y of step i-NSET has been read back
                e2e_compute(j, stream=s_cmp)
                ev_cmp[i].record(s_cmp)
            with torch.cuda.stream(s_out):
                s_out.wait_event(ev_cmp[i])
                y_p[j].copy_(y_d.view(torch.int16), non_blocking=True)
                ev_out[i].record(s_out)
        end.record(s_out)
        return start, end

    e2e_pipeline(args.warmup)
    torch.cuda.synchronize()
    barrier(world)
    e_start, e_end = e2e_pipeline(args.steps)
    torch.cuda.synchronize()
    e2e_ms = e_start.elapsed_time(e_end) / args.steps
    e2e_ms = max_over_ranks(e2e_ms, world)
    y_check = sets[(args.steps - 1) % NSET][4].view(torch.int16).cpu()
    e2e_y_ok = bool(torch.equal(y_p[(args.steps - 1) % NSET], y_check))
    h2d = scores_h.nbytes + q_h.nbytes + k_h.nbytes + v_h.nbytes
    d2h = y.numel() * 2

    def copy_ms(pairs, n):
        """Mean time of one round of the given copies alone, on a stream of their own."""
        s = torch.cuda.Stream(dev)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(s):
            for i in range(n + 2):
                if i == 2:
                    a.record(s)
                for dst, src in pairs:
                    dst.copy_(src, non_blocking=True)
            b.record(s)
        torch.cuda.synchronize()
        return a.elapsed_time(b) / n

    # the host link alone, with the same buffers and bytes as a step's copies: the floor under e2e
    h2d_ms = copy_ms(list(zip(sets[0][:4], (scores_p, q_p, k_p, v_p))), args.steps)
    d2h_ms = copy_ms([(y_p[0], sets[0][4].view(torch.int16))], args.steps)
    host_link = {"h2d_ms_per_step": h2d_ms, "d2h_ms_per_step": d2h_ms, "h2d_gbs": h2d / (h2d_ms * 1e-3) / 1e9,
                 "d2h_gbs": d2h / (d2h_ms * 1e-3) / 1e9,
                 "note": "the step's pinned copies timed alone (CUDA events on their own stream); the pipelined e2e "
                         "step cannot be shorter than the longer direction"}

    peak_tf = pk["bf16_tflops"]
    achieved = flops / (attn_ms * 1e-3) / 1e12
    traffic = ncu_traffic()
    line = {
        "metric": METRIC,
        "value": world * flops / (step_ms * 1e-3) / 1e12,
        "unit": "TFLOP/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": step_ms,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic",
        "config": {"workload": wl.name, "B": B, "T": T, "H": H, "K": K, "d_head": d, "group": g,
                   "rope_base": wl.base, "parallelism": f"replicas{world}",
                   "l2": "flushed before every timed step (2 GB write)", "seed": wl.seed,
                   "c_attn": acc.interaction_count(n_seg, g), "flops_per_step": flops,
                   "cv2_mean": float(np.mean([acc.cv2(n_seg[b * wl.Hr:(b + 1) * wl.Hr]) for b in range(B)]))},
        "step_ms_stats": stats(step_times),
        "stages_ms": {"route": stats(stage[:, 0]), "rope_pack_plan": stats(stage[:, 1]),
                      "attention": stats(stage[:, 2]), "note": "separate pass, an event between stages (no overlap)"},
        "rope_variants": rope_variants,
        "roofline": {"kernel": "attn_fwd_kernel<128>", "bound": "tensor", "achieved": achieved, "peak": peak_tf,
                     "unit": "TFLOP/s", "frac": achieved / peak_tf, "traffic": traffic,
                     "frac_sustained": achieved / pk.get("bf16_tflops_sustained", peak_tf),
                     "peak_source": f"{pk_kind} bf16 dense (burst); frac_sustained against the sustained figure",
                     "algorithmic": "4 * d_head * C_attn flops per launch (exact causal pairs)"},
        "e2e": {"value": world * flops / (e2e_ms * 1e-3) / 1e12, "unit": "TFLOP/s", "ms_per_step": e2e_ms,
                "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
                "api": "namoh_route + namoh_prefill from pinned host buffers, y copied back",
                "pipeline": f"host->device copies, compute and device->host copies on three streams, consecutive "
                            f"steps overlapped; {NSET} rotating device input/output sets ({NSET} x 51 MB > L2), "
                            f"no flush", "y_readback_matches_device": e2e_y_ok, "host_link": host_link},
        # per step: route (2 kernels) + RoPE/plan (1) + attention (1), in each of the three timed
        # passes (headline, stage breakdown, end to end), and one RoPE/plan launch per timed
        # step in each of the four RoPE variants
        "gpu_launches": 4 * 3 * args.steps + 4 * args.steps,
        "wall_s_timed_region": wall,
        "host_enqueue_ms_max": 1e3 * max(enqueue_s), "flush_ms_min": min(flush_ms), "stage_timing_gapless": gapless,
        "device_status": st,
    }

    if not args.no_configs:
        line["configs"] = run_configs(args, dev, pk, pk_kind)
        line["gpu_launches"] += line["configs"].pop("launches")
    if not args.no_decode:
        line["decode"] = run_decode(args, dev, pk, pk_kind)
        line["gpu_launches"] += line["decode"].pop("launches")
    if not args.no_layer:
        line["layer"] = run_layer(args, dev, pk, pk_kind)
        line["gpu_launches"] += line["layer"].pop("launches")
        line["shared_heads"] = run_shared(args, dev, pk, pk_kind)
        line["gpu_launches"] += line["shared_heads"].pop("launches")
        line["sa_namoh"] = run_sa(args, dev, pk, pk_kind)
        line["gpu_launches"] += line["sa_namoh"].pop("launches")
    clocks.__exit__(None, None, None)
    line["clocks"] = clocks.summary()
    return line


# The other prefill workloads: each is a parity case of the tests and is measured here as its own
# section (the headline stays on the balanced workload).
CONFIG_WORKLOADS = (ni.PR1, ni.SKEWED, *ni.H_SWEEP, ni.GQA)


def run_configs(args, dev, pk, pk_kind):
    """Every other prefill workload: route, RoPE + plan and attention timed apart (an event between
    stages) and as whole steps, the L2 flushed before each; the attention kernel against the bf16
    peaks; routing and RoPE against HBM; the per-token KV accesses of App. B.5 (C_attn / T in
    prefill, Eq. app-routed-interactions; A_KV(T) of the last token, Eq. app-routed-kv); and the
    oracle timed on the host cores on the same workload."""
    import torch

    import paper_2609_38832_gb300 as namoh

    flush = torch.empty(2 << 30, dtype=torch.uint8, device=dev)
    up = lambda b: torch.from_numpy(np.ascontiguousarray(b).view(np.int16)).to(dev).view(torch.bfloat16)  # noqa: E731
    out = {"peak_source": f"{pk_kind} bf16 dense: burst {pk['bf16_tflops']}, sustained "
                          f"{pk.get('bf16_tflops_sustained')} TFLOP/s; HBM {pk['hbm_gbs']} GB/s",
           "l2": "flushed before every timed step (2 GB write)"}
    launches = 0
    for wl in CONFIG_WORKLOADS:
        B, T, H, K, d, g = wl.B, wl.T, wl.H, wl.K, wl.d, wl.g
        scores_h = wl.scores()
        q_h, k_h, v_h = wl.qkv()
        scores = torch.from_numpy(scores_h).to(dev)
        q, k, v = up(q_h), up(k_h), up(v_h)
        ws = namoh.Workspace()
        status = torch.zeros(1, dtype=torch.int32, device=dev)
        ro = namoh.namoh_route(scores, wl.Kr, workspace=ws, status=status)
        q_rot, k_cache = torch.empty_like(q), torch.empty_like(k)
        plan = namoh.namoh_attention_plan(ro.seg_offsets, B=B, T=T, H=H, K=K, group=g)
        y = torch.empty((B, T, K, d), dtype=torch.bfloat16, device=dev)
        stages = (
            lambda: namoh.namoh_route(scores, wl.Kr, workspace=ws, status=status, out=ro),
            lambda: namoh.namoh_rope_pack(q, k, v, ro.seg_offsets, B=B, T=T, H=H, K=K, group=g, rope_base=wl.base,
                                          q_rot=q_rot, k_cache=k_cache, v_cache=v, status=status, plan=plan),
            lambda: namoh.namoh_attention(q_rot, k_cache, v, ro.seg_offsets, ro.row_src, ro.gate, plan, B=B, T=T,
                                          H=H, K=K, group=g, y=y, status=status),
        )
        whole = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]
        parts = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(args.steps)]
        for i in range(args.warmup + args.steps):  # whole steps (kernels overlap by programmatic launch)
            flush.fill_(i & 0xFF)
            if i >= args.warmup:
                whole[i - args.warmup][0].record()
            for f in stages:
                f()
            if i >= args.warmup:
                whole[i - args.warmup][1].record()
        for i in range(args.steps):  # the stage breakdown
            flush.fill_(i & 0xFF)
            for j, f in enumerate(stages):
                parts[i][j].record()
                f()
            parts[i][3].record()
        torch.cuda.synchronize()
        launches += 2 * args.steps * 4  # route 2 + RoPE/plan 1 + attention 1, in both passes
        step_t = [a.elapsed_time(b) for a, b in whole]
        st_t = np.array([[parts[i][j].elapsed_time(parts[i][j + 1]) for j in range(3)] for i in range(args.steps)])
        seg = ro.seg_offsets.cpu().numpy()
        n_seg = acc.segment_lengths(seg)
        flops = acc.attention_flops(n_seg, d, g)
        c_attn = acc.interaction_count(n_seg, g)
        top = ro.topk_head.cpu().numpy()
        a_kv = [acc.kv_activation(n_seg[b * wl.Hr:(b + 1) * wl.Hr], top[b, T - 1]) for b in range(B)]
        R = B * T * wl.Kr
        rbytes = acc.route_bytes(B, T, wl.Hr, wl.Kr)
        pbytes = acc.rope_pack_bytes(R, d, g, copy_v=False)
        attn_mean = float(st_t[:, 2].mean())
        achieved = flops / (attn_mean * 1e-3) / 1e12
        gbs = lambda nbytes, ms: nbytes / (ms * 1e-3) / 1e9  # noqa: E731
        entry = {
            "shape": {"B": B, "T": T, "H": H, "K": K, "d_head": d, "group": g, "rope_base": wl.base,
                      "zipf_bias": wl.zipf_bias, "seed": wl.seed},
            "segments": {"n_max": int(n_seg.max()), "n_min": int(n_seg.min()),
                         "cv2_mean": float(np.mean([acc.cv2(n_seg[b * wl.Hr:(b + 1) * wl.Hr]) for b in range(B)]))},
            "c_attn": c_attn, "flops": flops,
            "kv_accesses_per_token_prefill": c_attn / (B * T),
            "a_kv_last_token": float(np.mean(a_kv)),
            "kv_storage_per_sequence": int(acc.kv_storage(n_seg)) // B,
            "step_ms": stats(step_t), "step_tflops": flops / (np.median(step_t) * 1e-3) / 1e12,
            "route": {"ms": stats(st_t[:, 0]), "bytes": rbytes, "hbm_gbs": gbs(rbytes, st_t[:, 0].mean()),
                      "frac_measured_hbm": gbs(rbytes, st_t[:, 0].mean()) / pk["hbm_gbs"]},
            "rope_pack_plan": {"ms": stats(st_t[:, 1]), "bytes": pbytes, "hbm_gbs": gbs(pbytes, st_t[:, 1].mean()),
                               "frac_measured_hbm": gbs(pbytes, st_t[:, 1].mean()) / pk["hbm_gbs"]},
            "roofline": {"kernel": f"attn_fwd_kernel<{d}>", "bound": "tensor", "achieved": achieved,
                         "peak": pk["bf16_tflops"], "unit": "TFLOP/s", "frac": achieved / pk["bf16_tflops"],
                         "frac_sustained": achieved / pk.get("bf16_tflops_sustained", pk["bf16_tflops"]),
                         "ms": stats(st_t[:, 2])},
            "device_status": int(status.item()),
        }
        if not args.no_cpu_baseline:
            cb = oracle_prefill_sample(wl, min_seconds=3.0)
            entry["cpu_baseline"] = {k_: cb[k_] for k_ in ("value", "unit", "cores", "kind", "sample")}
            entry["cpu_baseline"]["seconds_per_step"] = cb["seconds_per_step"]
        out[wl.name] = entry
        del scores, q, k, v, q_rot, k_cache, y, ro, plan, ws
        torch.cuda.empty_cache()
    out["launches"] = launches
    return out


LAYER_D_MODEL = 2048  # the paper's model width (its experiments fix 2048)


def run_layer(args, dev, pk, pk_kind):
    """The balanced workload as a whole attention layer at d_model = 2048: the sparse QKV
    projection (Eq. namoh-qkv), routing, RoPE + routed attention + combine, and the output
    projection (Eq. namoh-attention), random bf16 weights.  Each stage and the whole step are
    timed with the L2 flushed before every timed launch sequence."""
    import torch

    import paper_2609_38832_gb300 as namoh

    wl = ni.BALANCED
    B, T, H, K, d, g = wl.B, wl.T, wl.H, wl.K, wl.d, wl.g
    Hr, Kr = H // g, K // g
    d_model = LAYER_D_MODEL
    N, R = B * T, B * T * Kr
    gen = torch.Generator(device=dev)
    gen.manual_seed(wl.seed)
    x = torch.randn((N, d_model), generator=gen, device=dev).to(torch.bfloat16)
    w_qkv = (torch.randn((Hr, (g + 2) * d, d_model), generator=gen, device=dev) / d_model ** 0.5).to(torch.bfloat16)
    w_o = (torch.randn((Hr, d_model, g * d), generator=gen, device=dev) / (g * d) ** 0.5).to(torch.bfloat16)
    scores = torch.from_numpy(wl.scores()).to(dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    ws_r, ws_p, ws_l = namoh.Workspace(), namoh.Workspace(), namoh.Workspace()
    ro = namoh.namoh_route(scores, Kr, workspace=ws_r, status=status)
    q = torch.empty((R * g, d), dtype=torch.bfloat16, device=dev)
    k = torch.empty((R, d), dtype=torch.bfloat16, device=dev)
    v = torch.empty((R, d), dtype=torch.bfloat16, device=dev)
    k_cache = torch.empty_like(k)
    y = torch.empty((B, T, K, d), dtype=torch.bfloat16, device=dev)
    o = torch.empty((N, d_model), dtype=torch.float32, device=dev)
    flush = torch.empty(2 << 30, dtype=torch.uint8, device=dev)

    def qkv():
        namoh.namoh_proj_qkv(x, w_qkv, ro.seg_offsets, ro.row_src, B=B, H=H, K=K, group=g, q=q, k=k, v=v,
                             workspace=ws_l, status=status)

    def out():
        namoh.namoh_proj_out(y, w_o, ro.seg_offsets, ro.row_src, B=B, H=H, K=K, group=g, o=o, workspace=ws_l,
                             status=status)

    def step():
        namoh.namoh_route(scores, Kr, workspace=ws_r, status=status, out=ro)
        qkv()
        namoh.namoh_prefill(q, k, v, ro.seg_offsets, ro.row_src, ro.gate, B=B, T=T, H=H, K=K, group=g,
                            rope_base=wl.base, y=y, k_cache=k_cache, workspace=ws_p, status=status)
        out()

    def timed(fn):
        evs = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]
        for i in range(args.warmup + args.steps):
            flush.fill_(i & 0xFF)
            if i >= args.warmup:
                evs[i - args.warmup][0].record()
            fn()
            if i >= args.warmup:
                evs[i - args.warmup][1].record()
        torch.cuda.synchronize()
        return float(np.mean([a.elapsed_time(b) for a, b in evs]))

    step()
    torch.cuda.synchronize()
    # the output projection runs one product-and-combine pair per token chunk of at most 1 GB of
    # bf16 per-slot products (the library's chunking); a projection over one chunk of a small
    # layout builds its tile list inside the GEMM, otherwise two list kernels run first
    out_chunk = min(N, max(128, (1 << 30) // (Kr * d_model * 2)))
    nchunk = -(-N // out_chunk)
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    nseg = B * Hr
    list_in_kernel = nseg <= 1024 and -(-(-(-R // 128) + nseg) // sms) <= 288
    qkv_launches = 1 if list_in_kernel else 3
    out_launches = 2 * nchunk + (0 if (list_in_kernel and nchunk == 1) else 2)
    n_seg = acc.segment_lengths(ro.seg_offsets.cpu().numpy())
    f_attn = acc.attention_flops(n_seg, d, g)
    f_qkv = 2.0 * R * d_model * (g + 2) * d
    f_out = 2.0 * R * g * d * d_model
    ms_qkv, ms_out, ms_step = timed(qkv), timed(out), timed(step)
    peak = pk["bf16_tflops"]
    tf = lambda f, ms: f / (ms * 1e-3) / 1e12  # noqa: E731
    return {
        "workload": f"{wl.name} with d_model={d_model}, random bf16 weights",
        "qkv_projection": {"ms": ms_qkv, "tflops": tf(f_qkv, ms_qkv), "frac_bf16": tf(f_qkv, ms_qkv) / peak,
                           "flops": f_qkv, "kernel": "proj_kernel (tcgen05, rows gathered by cp.async)"},
        "out_projection": {"ms": ms_out, "tflops": tf(f_out, ms_out), "frac_bf16": tf(f_out, ms_out) / peak,
                           "flops": f_out, "kernel": "proj_kernel, per-slot products (bf16), then combine_kernel (fp32 sums)"},
        "layer_step": {"ms": ms_step, "tflops": tf(f_qkv + f_attn + f_out, ms_step),
                       "frac_bf16": tf(f_qkv + f_attn + f_out, ms_step) / peak,
                       "flops": f_qkv + f_attn + f_out,
                       "stages": "route, QKV projection, RoPE + attention + combine, output projection"},
        "peak_source": f"{pk_kind} bf16 dense (burst)",
        "l2": "flushed before every timed launch sequence (2 GB write)",
        "device_status": int(status.item()),
        # timed launches: QKV, OUT (a GEMM and a combine per chunk, after the list kernels when
        # they run), and the step (route 2 + QKV + prefill 2 + OUT)
        "launches": args.steps * (qkv_launches + out_launches + (2 + qkv_launches + 2 + out_launches)),
    }


def run_shared(args, dev, pk, pk_kind):
    """Shared heads at the balanced workload's sizes (B4 T4096 d128), Hs = 4: the paper's
    sliding window of 128 tokens and the full causal prefix (namoh_shared_prefill), L2 flushed
    before every timed launch.  Flops: 4 d per causal (query, key) pair inside the window."""
    import torch

    import paper_2609_38832_gb300 as namoh

    B, T, Hs, d = 4, 4096, 4, 128
    gen = torch.Generator(device=dev)
    gen.manual_seed(7)
    q, k, v = (torch.randn((B, Hs, T, d), generator=gen, device=dev).to(torch.bfloat16) for _ in range(3))
    y = torch.empty((B, T, Hs, d), dtype=torch.bfloat16, device=dev)
    k_cache = torch.empty((B * Hs * T, d), dtype=torch.bfloat16, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    ws = namoh.Workspace()
    flush = torch.empty(2 << 30, dtype=torch.uint8, device=dev)
    out = {"workload": f"B{B} T{T} Hs{Hs} d{d}, bf16 N(0,1) inputs", "peak_source": f"{pk_kind} bf16 dense (burst)"}
    for name, window in (("window_128", 128), ("full_prefix", 0)):
        def run():
            namoh.namoh_shared_prefill(q, k, v, window=window, y=y, k_cache=k_cache, workspace=ws, status=status)

        evs = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]
        for i in range(args.warmup + args.steps):
            flush.fill_(i & 0xFF)
            if i >= args.warmup:
                evs[i - args.warmup][0].record()
            run()
            if i >= args.warmup:
                evs[i - args.warmup][1].record()
        torch.cuda.synchronize()
        ms = float(np.mean([a.elapsed_time(b) for a, b in evs]))
        pairs = B * Hs * sum(min(t + 1, window) if window else t + 1 for t in range(T))
        flops = 4.0 * d * pairs
        tf = flops / (ms * 1e-3) / 1e12
        out[name] = {"ms": ms, "tflops": tf, "frac_bf16": tf / pk["bf16_tflops"], "flops": flops}
    out["device_status"] = int(status.item())
    out["launches"] = 2 * args.steps * 3  # layout, RoPE + plan, attention per call
    return out


def run_sa(args, dev, pk, pk_kind):
    """SA + NAMOH (namoh_sa_prefill) on the balanced workload: 32-key blocks, alpha = 1/5, L2 flushed
    before every timed call, beside the dense routed prefill on the same routing.  Flops: 4 d per
    attended (query, key) pair, sum over heads of Phi_{alpha,B}(n_i) (App. B.3 Eq.
    app-fractional-causal-sum); the kernel still runs every causal key tile and masks the blocks a
    query does not keep, so its time is the dense prefill's plus the selection."""
    import torch

    import paper_2609_38832_gb300 as namoh

    wl = ni.BALANCED
    block, num, den = 32, 1, 5
    ro = namoh.namoh_route(torch.from_numpy(wl.scores()).to(dev), wl.Kr)
    qh, kh, vh = wl.qkv()
    up = lambda b: torch.from_numpy(b.view(np.int16)).to(dev).view(torch.bfloat16)
    q, k, v = up(qh), up(kh), up(vh)
    kw = dict(B=wl.B, T=wl.T, H=wl.H, K=wl.K, group=wl.g, rope_base=wl.base)
    y = torch.empty((wl.B, wl.T, wl.K, wl.d), dtype=torch.bfloat16, device=dev)
    k_cache = torch.empty_like(k)
    mask = torch.empty((k.shape[0] * wl.g, namoh._abi.load().namoh_sa_mask_words(wl.T, block)), dtype=torch.int32,
                       device=dev)
    ws_sa, ws_dense = namoh.Workspace(), namoh.Workspace()
    flush = torch.empty(2 << 30, dtype=torch.uint8, device=dev)
    calls = {
        "sa": lambda: namoh.namoh_sa_prefill(q, k, v, ro.seg_offsets, ro.row_src, ro.gate, block=block,
                                             alpha_num=num, alpha_den=den, y=y, sa_mask=mask, k_cache=k_cache,
                                             workspace=ws_sa, status=ro.status, **kw),
        "dense": lambda: namoh.namoh_prefill(q, k, v, ro.seg_offsets, ro.row_src, ro.gate, y=y, k_cache=k_cache,
                                             workspace=ws_dense, status=ro.status, **kw),
    }
    ms, ms_stats = {}, {}
    for name, run in calls.items():
        evs = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]
        for i in range(args.warmup + args.steps):
            flush.fill_(i & 0xFF)
            if i >= args.warmup:
                evs[i - args.warmup][0].record()
            run()
            if i >= args.warmup:
                evs[i - args.warmup][1].record()
        torch.cuda.synchronize()
        ms[name] = float(np.mean([a.elapsed_time(b) for a, b in evs]))
        ms_stats[name] = stats([a.elapsed_time(b) for a, b in evs])
    n = np.diff(ro.seg_offsets.cpu().numpy()).astype(np.int64)
    pairs_sa = 0
    for ni_ in n:
        r = np.arange(1, ni_ + 1, dtype=np.int64)
        nb = (r + block - 1) // block
        kept = (nb * num + den - 1) // den
        pairs_sa += int(np.sum(r - block * (nb - kept)))  # a_{alpha,B}(r), Eq. app-selected-entries
    pairs_dense = int(np.sum(n * (n + 1) // 2))
    # key tiles of 128 that some query of a 128-row tile keeps (a kept block, or its own block): the
    # fraction of the causal tiles a tile-skipping kernel could leave out is 1 minus this
    m = mask.cpu().numpy().view(np.uint32)
    seg = ro.seg_offsets.cpu().numpy().astype(np.int64)
    need, total = 0, 0
    for s_ in range(len(seg) - 1):
        nn = int(seg[s_ + 1] - seg[s_])
        for qt in range((nn + 127) // 128):
            rows = np.arange(qt * 128, min(nn, qt * 128 + 128))
            words = np.bitwise_or.reduce(m[seg[s_] + rows], axis=0)
            bits = np.unpackbits(words.view(np.uint8), bitorder="little")
            for kv in range(qt):  # the diagonal tile is always needed
                total += 1
                need += int(bits[kv * 128 // block:(kv + 1) * 128 // block].any())
    tiles_needed = need / total if total else 1.0
    flops_sa = 4.0 * wl.d * wl.g * pairs_sa
    tf = flops_sa / (ms["sa"] * 1e-3) / 1e12
    return {"workload": f"{wl.name}, blocks of {block}, alpha {num}/{den}", "ms": ms["sa"],
            "dense_prefill_ms": ms["dense"], "sa_pairs_over_dense": pairs_sa / pairs_dense,
            "off_diagonal_key_tiles_needed": tiles_needed, "ms_stats": ms_stats,
            "tflops_attended": tf, "frac_bf16": tf / pk["bf16_tflops"], "flops_attended": flops_sa,
            "peak_source": f"{pk_kind} bf16 dense (burst)", "device_status": int(ro.status.item()),
            # per timed pair: SA (RoPE + plan, pooling, selection, attention) and dense (RoPE + plan, attention)
            "launches": args.steps * (4 + 2),
            "note": "every causal key tile is computed; blocks not kept are masked in the softmax"}


def run_decode(args, dev, pk, pk_kind):
    import torch

    import paper_2609_38832_gb300 as namoh

    wl = ni.DECODE
    B, Hr, Kr, d, g = wl.B, wl.Hr, wl.Kr, wl.d, wl.g
    steps = args.decode_steps
    # a shorter prefix only for small profiler captures; the timed workload is the full one
    prefix = args.decode_prefix or wl.prefix
    s = torch.from_numpy(ni.router_scores(wl.seed, B, prefix, Hr)).to(dev)
    ws = namoh.Workspace()
    ro = namoh.namoh_route(s, Kr, workspace=ws)
    torch.cuda.synchronize()
    # routing of the prefix: HBM-bound, measured here (5 repetitions)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(6)]
    for i in range(5):
        ev[i].record()
        namoh.namoh_route(s, Kr, workspace=ws, out=ro)
    ev[5].record()
    torch.cuda.synchronize()
    route_ms = ev[0].elapsed_time(ev[5]) / 5
    # the same routing with loss-free balancing biases (selection on a + b, gates a)
    bias = torch.from_numpy((np.random.default_rng(wl.seed).standard_normal(Hr) * 0.02 / Hr).astype(np.float32)).to(dev)
    namoh.namoh_route(s, Kr, workspace=ws, out=ro, bias=bias)
    ev[0].record()
    for i in range(5):
        namoh.namoh_route(s, Kr, workspace=ws, out=ro, bias=bias)
    ev[5].record()
    torch.cuda.synchronize()
    route_biased_ms = ev[0].elapsed_time(ev[5]) / 5
    route_bytes = acc.route_bytes(B, prefix, Hr, Kr)
    seg = ro.seg_offsets.cpu().numpy().astype(np.int64)
    del s, ro
    torch.cuda.empty_cache()
    nseg = B * Hr
    n = seg[1:] - seg[:-1]
    head = steps + args.warmup
    seg_base = seg[:-1] + np.arange(nseg) * head
    cap = (n + head).astype(np.int32)
    rows = int(seg[-1] + nseg * head)
    gen = torch.Generator(device=dev)
    gen.manual_seed(wl.seed)
    kc = torch.randn((rows, d), generator=gen, device=dev, dtype=torch.bfloat16)
    vc = torch.randn((rows, d), generator=gen, device=dev, dtype=torch.bfloat16)
    seg_len = torch.from_numpy(n.astype(np.int32)).to(dev)
    sb, cp = torch.from_numpy(seg_base).to(dev), torch.from_numpy(cap).to(dev)
    sc_h, q_h, k_h, v_h = ni.decode_step_inputs(wl.seed, head, B, Hr, Kr, d, g)
    # the oracle's sample (sequences 0 .. DECODE_CPU_SEQS - 1, every step): their seeded prefix
    # rows, copied before any decode step appends to the cache
    cpu_seqs = 0 if args.no_cpu_baseline else min(DECODE_CPU_SEQS, B)
    cpu_state = None
    if cpu_seqs:
        segs = np.arange(cpu_seqs * Hr)
        o_cap = (n[segs] + steps).astype(np.int32)
        o_base = np.concatenate([[0], np.cumsum(o_cap)[:-1]]).astype(np.int64)
        o_kc = np.zeros((int(o_cap.sum()), d))
        o_vc = np.zeros((int(o_cap.sum()), d))
        for s_ in segs:
            lo, m = int(seg_base[s_]), int(n[s_])
            o_kc[o_base[s_]:o_base[s_] + m] = kc[lo:lo + m].float().cpu().numpy()
            o_vc[o_base[s_]:o_base[s_] + m] = vc[lo:lo + m].float().cpu().numpy()
        cpu_state = (o_kc, o_vc, o_base, n[segs].astype(np.int32), o_cap)
    sc = torch.from_numpy(sc_h[:, :, None, :].copy()).to(dev)
    qd = torch.from_numpy(q_h.view(np.int16)).to(dev).view(torch.bfloat16)
    kd = torch.from_numpy(k_h.view(np.int16)).to(dev).view(torch.bfloat16)
    vd = torch.from_numpy(v_h.view(np.int16)).to(dev).view(torch.bfloat16)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    dws = namoh.Workspace()
    y = torch.empty((B, Kr * g, d), dtype=torch.bfloat16, device=dev)
    rt = namoh.namoh_route(sc[0], Kr, compact=False, workspace=dws, status=status)

    def dstep(t, e=None):
        if e is not None:
            e[0].record()
        namoh.namoh_route(sc[t], Kr, compact=False, workspace=dws, status=status, out=rt)
        if e is not None:
            e[1].record()
        namoh.namoh_decode(rt.topk_head.view(B, Kr), rt.gate.view(B, Kr), qd[t], kd[t], vd[t], H=wl.H, K=wl.K,
                           group=g, rope_base=wl.base, k_cache=kc, v_cache=vc, seg_base=sb, seg_len=seg_len,
                           seg_cap=cp, y=y, workspace=dws, status=status)
        if e is not None:
            e[2].record()

    for t in range(args.warmup):
        dstep(t)
    torch.cuda.synchronize()
    lens_before = seg_len.cpu().numpy().astype(np.int64)
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(steps)]
    tops = []
    for t in range(steps):
        dstep(args.warmup + t, evs[t])
        tops.append(rt.topk_head.view(B, Kr).clone())
    torch.cuda.synchronize()
    times = np.array([[e[0].elapsed_time(e[1]), e[1].elapsed_time(e[2])] for e in evs])
    # algorithmic bytes per step from the lengths each step attended over
    lens = lens_before.copy()
    total_bytes = 0
    for t in range(steps):
        top = tops[t].cpu().numpy()
        segs = (np.arange(B)[:, None] * Hr + top).reshape(-1)
        after = lens[segs] + 1
        total_bytes += acc.decode_bytes(after, d, g)
        lens[segs] = after
    assert np.array_equal(lens, seg_len.cpu().numpy()), "decode lengths diverged from the bookkeeping"
    step_ms = float(np.median(times.sum(1)))
    decode_ms = float(times[:, 1].mean())  # HBM GB/s divides by the kernel's average duration
    bytes_per_step = total_bytes / steps
    gbs = bytes_per_step / (decode_ms * 1e-3) / 1e9
    out = {
        "workload": wl.name if prefix == wl.prefix else f"{wl.name} at prefix {prefix} (profiling size)",
        "steps": steps, "tokens_per_s": B / (step_ms * 1e-3), "ms_per_step": step_ms,
        "step_ms_stats": stats(times.sum(1)), "decode_ms_stats": stats(times[:, 1]),
        "route_ms": float(times[:, 0].mean()), "decode_ms": decode_ms, "bytes_per_step": bytes_per_step,
        "hbm_gbs": gbs, "frac_measured_hbm": gbs / pk["hbm_gbs"], "frac_nominal_8tbs": gbs / NOMINAL_HBM_GBS,
        "hbm_peak_source": f"{pk_kind} copy bandwidth {pk['hbm_gbs']} GB/s",
        "prefix_route": {"ms": route_ms, "bytes": route_bytes, "hbm_gbs": route_bytes / (route_ms * 1e-3) / 1e9,
                         "frac_measured_hbm": route_bytes / (route_ms * 1e-3) / 1e9 / pk["hbm_gbs"]},
        "prefix_route_biased": {"ms": route_biased_ms, "hbm_gbs": route_bytes / (route_biased_ms * 1e-3) / 1e9,
                                "frac_measured_hbm": route_bytes / (route_biased_ms * 1e-3) / 1e9 / pk["hbm_gbs"],
                                "note": "selection on softmax affinities plus per-head biases (namoh_route_biased)"},
        "cache_gb": 2 * rows * d * 2 / 1e9, "device_status": int(status.item()),
        "launches": 4 * steps + 2 * 5 * 3,  # decode steps; 5 timed prefix routings of 3 kernels, plain and biased
    }
    del kc, vc
    torch.cuda.empty_cache()
    if cpu_state is not None:
        out["cpu_baseline"] = oracle_decode_sample(cpu_state, cpu_seqs, sc_h[args.warmup:], q_h[args.warmup:],
                                                   k_h[args.warmup:], v_h[args.warmup:], wl, steps)
    return out


DECODE_CPU_SEQS = 2  # sequences of the decode workload the oracle runs in the CPU baseline


def oracle_decode_sample(state, nseq, sc, q, k, v, wl, steps):
    """The oracle, as it stands, on sequences 0 .. nseq-1 of the decode workload for every step:
    routing of the new token and the decode step (append at rank, attend, gate)."""
    import oracle
    oracle.build()
    o_kc, o_vc, o_base, o_len, o_cap = state
    threads = oracle.default_threads()
    t0 = time.perf_counter()
    for t in range(steps):
        r = oracle.route(sc[t][:nseq, None, :], wl.Kr)
        oracle.decode_step(r["topk_head"][:, 0], r["gate"][:, 0], q[t][:nseq], k[t][:nseq], v[t][:nseq], wl.Hr,
                           wl.d, wl.g, wl.base, o_kc, o_vc, o_base, o_len, o_cap)
    sec = time.perf_counter() - t0
    return {"value": nseq * steps / sec, "unit": "tokens/s", "cores": threads, "kind": "oracle",
            "sample": f"sequences 0-{nseq - 1} of {wl.B} (their seeded 131072-token prefixes), all {steps} steps, "
                      f"route + decode step per token, {sec:.1f} s, fp64 C on {threads} host threads ({cpu_model()})",
            "seconds_per_step": sec / steps}


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    if world <= 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device="cuda")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["namoh", "reference"], default="namoh")
    ap.add_argument("--decode-steps", type=int, default=256)
    ap.add_argument("--decode-prefix", type=int, default=0,
                    help="routed prefix length of the decode section (0: the workload's 131072); smaller only "
                         "for profiler captures")
    ap.add_argument("--no-decode", action="store_true")
    ap.add_argument("--no-layer", action="store_true")
    ap.add_argument("--no-configs", action="store_true")
    ap.add_argument("--only", choices=["configs", "decode", "layer", "shared", "sa"], default=None,
                    help="run one section alone and print it (small profiler captures); not a bench line")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))

    if args.impl == "reference":
        # the reference arm is the fp64 oracle on the host cores; rank 0 only
        if rank != 0:
            return
        wl = ni.BALANCED
        for _ in range(args.warmup):  # untimed: the oracle's library load and first touch of the inputs
            oracle_prefill_sample(wl, min_seconds=0.0, max_reps=1)
        samples, t_start = [], time.perf_counter()
        for _ in range(args.steps):  # each step: the whole workload once; stop after ~3 minutes
            samples.append(oracle_prefill_sample(wl, min_seconds=0.0, max_reps=1))
            if time.perf_counter() - t_start > 180.0:
                break
        val = float(np.mean([s_["value"] for s_ in samples]))
        cb = dict(samples[0])
        cb["value"] = val
        sec = float(np.mean([s_["seconds_per_step"] for s_ in samples]))
        print(json.dumps({
            "metric": METRIC, "value": val, "unit": "TFLOP/s", "n_gpus": world, "steps": len(samples),
            "warmup": args.warmup, "ms_per_step": sec * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None,
            "dtype": "f64", "data": "synthetic", "impl": "reference",
            "config": {"workload": wl.name, "B": wl.B, "T": wl.T, "H": wl.H, "K": wl.K, "d_head": wl.d},
            "cpu_baseline": {k_: cb[k_] for k_ in ("value", "unit", "cores", "kind", "sample")},
            "e2e": {"value": val, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        }))
        return

    if args.only:
        import torch
        dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", 0)))
        torch.cuda.set_device(dev)
        pk, pk_kind = peaks()
        fn = {"configs": run_configs, "decode": run_decode, "layer": run_layer, "shared": run_shared,
              "sa": run_sa}[args.only]
        if rank == 0:
            print(json.dumps({"section": args.only, args.only: fn(args, dev, pk, pk_kind)}))
        return
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    line = run_gpu(args, rank, world)
    if rank == 0 and not args.no_cpu_baseline:
        cb = oracle_prefill_sample(ni.BALANCED)
        line["cpu_baseline"] = {k_: cb[k_] for k_ in ("value", "unit", "cores", "kind", "sample")}
    if rank == 0:
        print(json.dumps(line))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
