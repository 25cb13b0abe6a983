#!/usr/bin/env python3
"""Throughput of the L_JAB hot path on GB300: candidate-loss evaluations per second.

One step = one forward L_JAB + STE/LSQ scale-gradient evaluation of the Mistral-7B-shaped attention
block (d_model 4096, 32 query / 8 KV heads of 128, RoPE theta 1e4), X = 128 sequences x 2048 tokens
of Student-t(4) unit-variance activations, 3-bit groups of 128: an iteration of the scale fit
(jab_loss_backward_scales_prepared). The teacher output A(X; W) and the fp16 copy of X are made once
before the timed region: both are shared by every evaluation on the same calibration batch, like
the fitting loop's 200 steps. Reported beside it: the forward-only rate (jab_loss_forward, one
candidate), the Fisher-coupling probe (loss and squared STE weight-gradient norm at 2 bits,
jab_loss_backward_weights), the end-to-end rate with host buffers, and under "workloads" the rates of
the other four workloads (GPT-2 smoke step, GPT-2 four-candidate scoring pass, the 32-block x 5-width
Mistral sensitivity table, the long-context Mistral fitting step), each with its roofline and CPU
oracle baseline.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference] [--workload NAME]

Under torchrun the ranks evaluate one batch sharded by sequence: rank r holds its own seeded shard of
the workload's size, and every step combines the shards' loss and scale gradient with one
all-reduce of 1 + D d/G fp64 values (weak scaling; value = shards evaluated by all ranks / max rank
time).
`--impl reference` times the float64 CPU oracle on a bounded sample of the same workload.
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

import numpy as np  # noqa: E402
import torch  # noqa: E402

from paper_2609_34866_gb300.multi import combine_shards, dist_env, max_over_ranks  # noqa: E402
from workloads import WORKLOADS, make_block_weights, make_x  # noqa: E402

METRIC = "JAB candidate-loss evals/s (fwd+STE bwd), Mistral-7B-shaped attention block"


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            m = json.load(f)
        return dict(hbm=float(m["hbm_gbs"]), bf16=float(m["bf16_tflops"]),
                    bf16_sus=float(m["bf16_tflops_sustained"]),
                    sm_max_mhz=float(m.get("sm_max_mhz", 2070.0)), source="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, sm_max_mhz=2070.0, source="fallback")


def work_of(wl, C=1):
    """Algorithmic FLOPs / bytes per launch site for one call over C candidates (GEMM = 2MNK;
    causal attention counts the lower triangle including the diagonal; backward attention = 2.5x
    forward; the KL term's two score products = the forward's two products; no dX GEMM). The
    quantiser reads W (2 B) and writes the fp16 operand (2 B) per weight, per candidate."""
    s = wl.shape
    N, D, d = wl.batch * wl.seq_len, s.d_out, s.d_model
    attn = 4.0 * wl.batch * s.n_q_heads * s.head_dim * wl.seq_len * (wl.seq_len + 1) / 2
    return {
        "proj_gemm": ("flop", 2.0 * N * C * D * d),
        "attn_fwd": ("flop", attn * C),
        "attn_kl": ("flop", attn * C),
        "attn_bwd": ("flop", 2.5 * attn),
        "wgrad_lsq": ("flop", 2.0 * N * D * d),
        "wgrad_store": ("flop", 2.0 * N * D * d),
        "attn_jvp": ("flop", 2.5 * attn * C),
        "convert_x": ("byte", 4.0 * N * d),
        "quantize": ("byte", 4.0 * D * d * C),
        "probe": ("byte", 2.0 * D * d * C),
    }


def roofline_of(sites, work_total, pk, sustained=True):
    """Roofline of the launch site with the largest summed device time: its algorithmic work over
    the timed region (work_total: site -> (kind, amount summed over the region)) divided by its
    summed device time, against the measured peak (sustained bf16 for a kernel inside a
    seconds-long loop)."""
    dom = max(sites, key=lambda k: sites[k][0])
    dom_ms, dom_ranges, _ = sites[dom]
    kind, amount = work_total.get(dom, ("flop", float("nan")))
    if kind == "flop":
        achieved = amount / (dom_ms / 1e3) / 1e12
        peak = pk["bf16_sus"] if sustained else pk["bf16"]
        bound, unit = "tensor", "TFLOP/s"
        note = (f"{pk['source']} {'sustained' if sustained else 'burst'} bf16 dense "
                f"(fp16 operands: same nominal rate)")
    else:
        achieved = amount / (dom_ms / 1e3) / 1e9
        bound, peak, unit = "hbm", pk["hbm"], "GB/s"
        note = f"{pk['source']} HBM copy bandwidth"
    return {"bound": bound, "achieved": achieved, "peak": peak, "unit": unit,
            "frac": achieved / peak, "kernel": dom, "launch_ms": dom_ms / max(1, dom_ranges),
            "peak_source": note}


def scaled_work(wl, C, times):
    """work_of(wl, C) with every amount multiplied by `times` (calls in the timed region)."""
    return {k: (kind, amt * times) for k, (kind, amt) in work_of(wl, C).items()}


def add_work(*ws):
    out = {}
    for w in ws:
        for k, (kind, amt) in w.items():
            out[k] = (kind, out.get(k, (kind, 0.0))[1] + amt)
    return out


def step_flops(wl):
    w = work_of(wl)
    fwd = w["proj_gemm"][1] + w["attn_fwd"][1]
    bwd = w["attn_bwd"][1] + w["wgrad_lsq"][1]
    return fwd, bwd


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons every 200 ms, during the timed region."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.rows = []
        self.proc = None
        sel = str(device_index)
        try:
            uuid = str(torch.cuda.get_device_properties(device_index).uuid)
            sel = uuid if uuid.startswith("GPU-") else "GPU-" + uuid
        except Exception:
            pass
        self.cmd = ["nvidia-smi", "-i", sel, f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                    "-lms", "200"]

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(self.cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL,
                                         text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None
        time.sleep(0.3)
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.rows.append([x.strip() for x in line.split(",")])

    def __exit__(self, *a):
        time.sleep(0.25)
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        sm, mx, reasons = [], [], set()
        for r in self.rows:
            try:
                sm.append(float(r[0]))
                mx.append(float(r[1]))
            except (ValueError, IndexError):
                continue
            for i, n in enumerate(names):
                if len(r) > 3 + i and r[3 + i].lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def config_of(wl):
    s = wl.shape
    return {"workload": wl.name, "batch": wl.batch, "seq_len": wl.seq_len, "d_model": s.d_model,
            "n_q_heads": s.n_q_heads, "n_kv_heads": s.n_kv_heads, "head_dim": s.head_dim,
            "rope": s.use_rope, "bits": list(wl.bits) if len(wl.bits) > 1 else wl.bits[0],
            "group_size": wl.group_size,
            "x": f"{wl.x_dist}" + (f"(df={wl.x_df})" if wl.x_df else "") +
                 (f", {wl.outlier_frac:.1%} channels x{wl.outlier_factor:g}" if wl.outlier_frac else ""),
            "scale_init": wl.scale_init,
            "l2": ("no flush: X (bf16) and A_ref (fp32) of every step are each larger than the 129 MB L2"
                   if wl.tokens * wl.shape.d_model * 2 > 129e6 else
                   "inputs smaller than L2: the step is launch- and latency-bound")}


def oracle_desc(wl):
    s = wl.shape
    return dict(d_model=s.d_model, n_q_heads=s.n_q_heads, n_kv_heads=s.n_kv_heads,
                head_dim=s.head_dim, group_size=wl.group_size, use_rope=s.use_rope,
                rope_theta=s.rope_theta, softmax_scale=0.0)


# ------------------------------------------------------------------------------------ oracle timing
def oracle_sample(wl, seqs=1):
    """The float64 oracle's fwd+STE-bwd on `seqs` sequences of the workload (teacher precomputed,
    as in the GPU step). Returns (seconds, description)."""
    from oracle import jab_oracle as O
    od = oracle_desc(wl)
    x = make_x(wl, batch=seqs).float().numpy().astype(np.float64)
    w = make_block_weights(wl).float().numpy().astype(np.float64)
    bits = wl.bits[0]
    scales = (O.init_scales_minmse(w, bits, wl.group_size) if wl.scale_init == "minmse"
              else O.init_scales_absmax(w, bits, wl.group_size))
    a_ref = O.block_forward(x, w, od)
    t0 = time.perf_counter()
    O.jab_loss_and_grad(x, w, scales, bits, od, a_ref=a_ref, kappa=0.0)
    dt = time.perf_counter() - t0
    return dt, (f"{seqs} of {wl.batch} sequences x {wl.seq_len} tokens, fwd + STE bwd, float64 "
                f"numpy oracle; evals/s extrapolated linearly in the number of sequences")


def oracle_fwd_sample(wl, seqs=1, block=0, with_teacher=False):
    """The float64 oracle's forward L_JAB for every candidate bit width of the workload on `seqs`
    sequences of block `block` (absmax scales), with its teacher pass timed too when
    with_teacher. Returns seconds."""
    from oracle import jab_oracle as O
    od = oracle_desc(wl)
    x = make_x(wl, batch=seqs).float().numpy().astype(np.float64)
    w = make_block_weights(wl, block).float().numpy().astype(np.float64)
    scales = [O.init_scales_absmax(w, b, wl.group_size) for b in wl.bits]
    t0 = time.perf_counter()
    a_ref = O.block_forward(x, w, od)
    t1 = time.perf_counter()
    for b, s_ in zip(wl.bits, scales):
        O.jab_loss(x, w, s_, b, od, a_ref=a_ref)
    t2 = time.perf_counter()
    return (t2 - t0) if with_teacher else (t2 - t1)


def run_reference(args, wl):
    world, rank, _ = dist_env()
    if rank != 0:
        return 0
    cores = os.cpu_count()
    times = []
    for i in range(args.warmup + args.steps):
        dt, sample = oracle_sample(wl, 1)
        if i >= args.warmup:
            times.append(dt)
    per_eval = statistics.mean(times) * wl.batch        # seconds per full-batch evaluation
    value = 1.0 / per_eval
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "evals/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": per_eval * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic", "config": config_of(wl),
            "cpu_baseline": {"value": value, "unit": "evals/s", "cores": cores, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": "evals/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------------------------------------------ our arm
def timed(J, fn, steps, warmup, st, barrier=lambda: None, sites=True):
    """Device time (ms) of `steps` calls of fn on stream st after `warmup` untimed calls, with CUDA
    events on the launching stream; with sites, also the per-launch-site device times."""
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    if sites:
        J.jab_timing_reset()
        J.jab_timing_enable(True)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    torch.cuda.synchronize()
    e0.record(st)
    for _ in range(steps):
        fn()
    e1.record(st)
    torch.cuda.synchronize()
    barrier()
    out = None
    if sites:
        J.jab_timing_enable(False)
        out = J.jab_timing_read()
    if J.jab_get_device_status() != 0:
        raise RuntimeError("device status set in a timed region")
    return e0.elapsed_time(e1), out


def timed_graph(J, fn, steps, warmup, st):
    """Device time (ms) of `steps` replays of a CUDA graph that holds one call of fn, with CUDA
    events on st (the replay stream). The library's calls launch only on the caller's stream and
    never synchronise the host, so one call captures whole; fn has run eagerly before."""
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        fn()
    for _ in range(max(warmup, 3)):
        graph.replay()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(st)
    for _ in range(steps):
        graph.replay()
    e1.record(st)
    torch.cuda.synchronize()
    if J.jab_get_device_status() != 0:
        raise RuntimeError("device status set in a timed region")
    return e0.elapsed_time(e1)


def rates(flops, ms_per_unit, pk):
    tf = flops / (ms_per_unit / 1e3) / 1e12
    return {"achieved_tflops": tf, "frac_of_bf16_peak": {"burst": tf / pk["bf16"],
                                                         "sustained": tf / pk["bf16_sus"],
                                                         "source": pk["source"]}}


def scales_for(J, desc, wl, W, bits, dev, mode=None):
    s = torch.empty((wl.shape.d_out, wl.shape.d_model // wl.group_size), dtype=torch.float32,
                    device=dev)
    if mode is None:
        mode = 1 if wl.scale_init == "minmse" else 0
    J.jab_init_scales(desc, bits, mode, W, s)
    return s


def wl_fit_step(J, wl, args, dev, pk, st, with_cpu):
    """A fwd + STE-bwd iteration of the scale fit (the calibration batch fixed: X converted once)."""
    B, T, bits = wl.batch, wl.seq_len, wl.bits[0]
    desc = J.desc_from_shape(wl.shape, wl.group_size)
    X = make_x(wl, device=dev)
    W = make_block_weights(wl, device=dev)
    s = scales_for(J, desc, wl, W, bits, dev)
    ws = J.Workspace(desc, B, T, 1, True, device=dev)
    A = torch.empty((B, T, wl.shape.n_q_heads * wl.shape.head_dim), dtype=torch.float32, device=dev)
    J.jab_reference_forward(desc, B, T, X, W, A, ws)
    J.jab_prepare_x(desc, B, T, X, ws)
    loss = torch.empty(1, dtype=torch.float64, device=dev)
    g = torch.empty_like(s)

    def fn():
        J.jab_loss_backward_scales_prepared(desc, B, T, X, W, A, bits, s, 0.0, loss, g, ws)

    steps = max(args.steps, 50 if wl.tokens < 65536 else 10)
    ms, _ = timed(J, fn, steps, args.warmup, st, sites=False)
    _, sites = timed(J, fn, steps, 1, st)
    fwd_f, bwd_f = step_flops(wl)
    out = {"metric": "fwd+STE-bwd evaluations/s (scale-fit iteration)", "value": steps / (ms / 1e3),
           "unit": "evals/s", "ms_per_eval": ms / steps, **rates(fwd_f + bwd_f, ms / steps, pk),
           "roofline": roofline_of(sites, scaled_work(wl, 1, steps), pk),
           "gpu_launches_per_eval": sum(v[2] for v in sites.values()) / steps,
           "config": config_of(wl)}
    if wl.tokens < 65536:
        # launch-bound: the same iteration replayed from a CUDA graph (host launch cost removed)
        gms = timed_graph(J, fn, steps, args.warmup, st)
        out["cuda_graph"] = {"value": steps / (gms / 1e3), "unit": "evals/s",
                             "ms_per_eval": gms / steps, **rates(fwd_f + bwd_f, gms / steps, pk)}
    if with_cpu:
        k = wl.batch if wl.tokens * wl.shape.d_model <= 4e6 else 1
        dt, _ = oracle_sample(wl, k)
        out["cpu_baseline"] = {"value": k / (dt * wl.batch), "unit": "evals/s",
                               "cores": os.cpu_count(), "kind": "oracle",
                               "sample": f"{k} of {wl.batch} sequences, fwd + STE bwd"
                                         + (", extrapolated linearly in sequences" if k < wl.batch else "")}
    return out


def wl_candidates(J, wl, args, dev, pk, st, with_cpu):
    """One forward L_JAB call over all candidate bit widths (one scoring pass of one block)."""
    B, T, C = wl.batch, wl.seq_len, len(wl.bits)
    desc = J.desc_from_shape(wl.shape, wl.group_size)
    X = make_x(wl, device=dev)
    W = make_block_weights(wl, device=dev)
    scales = [scales_for(J, desc, wl, W, b, dev) for b in wl.bits]
    ws = J.Workspace(desc, B, T, C, False, device=dev)
    A = torch.empty((B, T, wl.shape.n_q_heads * wl.shape.head_dim), dtype=torch.float32, device=dev)
    J.jab_reference_forward(desc, B, T, X, W, A, ws)
    loss = torch.empty(C, dtype=torch.float64, device=dev)

    def fn():
        J.jab_loss_forward(desc, B, T, X, W, A, list(wl.bits), scales, loss, ws)

    steps = max(args.steps, 20)
    ms, _ = timed(J, fn, steps, args.warmup, st, sites=False)
    _, sites = timed(J, fn, steps, 1, st)
    w = work_of(wl, C)
    flops = w["proj_gemm"][1] + w["attn_fwd"][1]
    out = {"metric": "candidate-loss evaluations/s (forward, all candidates in one call)",
           "value": C * steps / (ms / 1e3), "unit": "evals/s", "ms_per_call": ms / steps,
           "candidates_per_call": C, **rates(flops, ms / steps, pk),
           "roofline": roofline_of(sites, scaled_work(wl, C, steps), pk),
           "gpu_launches_per_call": sum(v[2] for v in sites.values()) / steps,
           "config": config_of(wl)}
    if with_cpu:
        k = 4
        dt = oracle_fwd_sample(wl, k)
        out["cpu_baseline"] = {"value": C * k / (dt * wl.batch), "unit": "evals/s",
                               "cores": os.cpu_count(), "kind": "oracle",
                               "sample": f"{k} of {wl.batch} sequences, forward of every candidate; "
                                         "extrapolated linearly in sequences"}
    return out


def wl_table(J, wl, args, dev, pk, st, with_cpu):
    """The whole sensitivity table: for each of the n_blocks seeded blocks, its teacher pass,
    absmax scales for every width and one forward over all widths (n_blocks x |bits| units)."""
    B, T, C, nb = wl.batch, wl.seq_len, len(wl.bits), wl.n_blocks
    desc = J.desc_from_shape(wl.shape, wl.group_size)
    X = make_x(wl, device=dev)
    Ws = [make_block_weights(wl, i, device=dev) for i in range(nb)]
    scales = [torch.empty((wl.shape.d_out, wl.shape.d_model // wl.group_size), dtype=torch.float32,
                          device=dev) for _ in wl.bits]
    ws = J.Workspace(desc, B, T, C, False, device=dev)
    A = torch.empty((B, T, wl.shape.n_q_heads * wl.shape.head_dim), dtype=torch.float32, device=dev)
    table = torch.empty((nb, C), dtype=torch.float64, device=dev)

    def fn():
        for i in range(nb):
            J.jab_reference_forward(desc, B, T, X, Ws[i], A, ws)
            for k, b in enumerate(wl.bits):
                J.jab_init_scales(desc, b, 0, Ws[i], scales[k])
            J.jab_loss_forward(desc, B, T, X, Ws[i], A, list(wl.bits), scales, table[i], ws)

    reps = 2
    ms, _ = timed(J, fn, reps, 1, st, sites=False)
    _, sites = timed(J, fn, 1, 0, st)
    w = add_work(scaled_work(wl, C, nb), scaled_work(wl, 1, nb))   # candidates + teacher passes
    flops = w["proj_gemm"][1] + w["attn_fwd"][1]
    out = {"metric": "(block, bit width) loss evaluations/s over the whole table, teacher passes "
                     "included", "value": nb * C * reps / (ms / 1e3), "unit": "evals/s",
           "ms_per_table": ms / reps, "units_per_table": nb * C, **rates(flops, ms / reps, pk),
           "roofline": roofline_of(sites, w, pk),
           "gpu_launches_per_table": sum(v[2] for v in sites.values()) + nb * C,
           "config": {**config_of(wl), "n_blocks": nb}}
    if with_cpu:
        dt = oracle_fwd_sample(wl, 1, with_teacher=True)
        out["cpu_baseline"] = {"value": C / (dt * wl.batch), "unit": "evals/s",
                               "cores": os.cpu_count(), "kind": "oracle",
                               "sample": f"block 0, 1 of {wl.batch} sequences, teacher + all "
                                         f"{C} widths; extrapolated linearly in sequences"}

    # The paper's own sensitivity score on the same blocks (Section 2.4, Eq. 5-6): the teacher pass
    # (A_ref and its log-sum-exp), a 10-probe Hutchinson trace through the forward-mode attention
    # kernel, and Omega C1 / C2 for every width.
    m, nbh = 10, 2
    lse = torch.empty((B, wl.shape.n_q_heads, T), dtype=torch.float32, device=dev)
    ws2 = J.Workspace(desc, B, T, 2, False, device=dev)
    wso = J.Workspace(desc, 1, 1, C, False, device=dev)
    trace = torch.empty(1, dtype=torch.float64, device=dev)
    c1, c2 = (torch.empty((nb, C), dtype=torch.float64, device=dev) for _ in range(2))

    def hutch():
        for i in range(nbh):
            J.jab_reference_forward(desc, B, T, X, Ws[i], A, ws2, lse=lse)
            J.jab_hutchinson_trace(desc, B, T, X, Ws[i], A, lse, m, 1000 + i, trace, ws2)
            for k, b in enumerate(wl.bits):
                J.jab_init_scales(desc, b, 0, Ws[i], scales[k])
            J.jab_omega_scores(desc, Ws[i], list(wl.bits), scales, trace, nb - 1 - i, c1[i], wso,
                               c2=c2[i])

    hms, _ = timed(J, hutch, 1, 1, st, sites=False)
    _, hsites = timed(J, hutch, 1, 0, st)
    w1 = work_of(wl, 1)   # per block: teacher (projection, attention), primal projection, m probes
    hw = {"proj_gemm": ("flop", w1["proj_gemm"][1] * nbh * (2 + m)),
          "attn_fwd": ("flop", w1["attn_fwd"][1] * nbh),
          "attn_jvp": ("flop", w1["attn_jvp"][1] * nbh * m),
          "convert_x": ("byte", w1["convert_x"][1] * nbh * 2),
          "quantize": ("byte", w1["quantize"][1] * nbh * 2),
          "probe": ("byte", w1["probe"][1] * nbh * m)}
    hflops = hw["proj_gemm"][1] + hw["attn_fwd"][1] + hw["attn_jvp"][1]
    out["hutchinson"] = {
        "metric": "blocks/s scored by the Hutchinson trace (10 probes) and Omega C1/C2 for every "
                  "width, teacher pass included", "value": nbh / (hms / 1e3), "unit": "blocks/s",
        "probe_evals_per_s": nbh * m / (hms / 1e3), "ms_per_block": hms / nbh,
        **rates(hflops / nbh, hms / nbh, pk), "roofline": roofline_of(hsites, hw, pk),
        "blocks_timed": nbh, "probes_per_block": m}
    return out


def measure_workloads(J, args, dev, pk, st, with_cpu):
    """Throughput of the other workloads (one line each; the headline stays the Mistral block)."""
    fns = {"gpt2_smoke": wl_fit_step, "gpt2_sweep": wl_candidates, "mistral_scoring": wl_table,
           "mistral_ste_long": wl_fit_step}
    out = {}
    for name, fn in fns.items():
        out[name] = fn(J, WORKLOADS[name], args, dev, pk, st, with_cpu)
        torch.cuda.empty_cache()
    return out


def run_ours(args, wl):
    import paper_2609_34866_gb300 as J
    from paper_2609_34866_gb300 import build as jb
    world, rank, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    dev = torch.device("cuda", torch.cuda.current_device())
    jb.build()
    pk = peaks()
    st = torch.cuda.current_stream()

    def barrier():
        if world > 1:
            torch.distributed.barrier()

    line = headline(J, args, wl, dev, pk, st, world, rank, barrier)
    workloads = None
    if world == 1 and not args.no_workloads and wl.name == "mistral_block" and args.batch is None:
        workloads = measure_workloads(J, args, dev, pk, st, not args.no_cpu_baseline)
    if world > 1:
        torch.distributed.destroy_process_group()
    if rank != 0:
        return 0
    if workloads is not None:
        line["workloads"] = workloads
    print(json.dumps(line), flush=True)
    return 0


def headline(J, args, wl, dev, pk, st, world, rank, barrier):
    """The headline step: one forward L_JAB + STE/LSQ scale-gradient evaluation of the workload
    (the scale-fit iteration: teacher and the fp16 copy of X made once per calibration batch)."""
    s = wl.shape
    B, T = wl.batch, wl.seq_len
    desc = J.desc_from_shape(s, wl.group_size)
    X = make_x(wl, device=dev, seed=wl.seed + rank)
    W = make_block_weights(wl, device=dev)
    bits = wl.bits[0]
    scales = scales_for(J, desc, wl, W, bits, dev)
    ws = J.Workspace(desc, B, T, 1, True, device=dev)
    A = torch.empty((B, T, s.n_q_heads * s.head_dim), dtype=torch.float32, device=dev)
    J.jab_reference_forward(desc, B, T, X, W, A, ws)
    J.jab_prepare_x(desc, B, T, X, ws)
    loss = torch.empty(1, dtype=torch.float64, device=dev)
    grad = torch.empty_like(scales)

    # Under torchrun the ranks evaluate one global batch of B * world sequences, sharded by
    # sequence (rank r holds its own seeded B sequences): every step combines the shards' loss and
    # scale gradient into the global ones with one all-reduce (multi.combine_shards).
    def step():
        J.jab_loss_backward_scales_prepared(desc, B, T, X, W, A, bits, scales, 0.0, loss, grad, ws)
        if world > 1:
            combine_shards(loss, grad, B, B * world)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if J.jab_get_device_status() != 0:
        raise RuntimeError("device status set during warm-up")

    # ---- timed region: K steps, device-timed with CUDA events on the launching stream
    J.jab_timing_reset()
    J.jab_timing_enable(True)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    torch.cuda.synchronize()
    with ClockSampler(dev.index) as clk:
        e0.record(st)
        for _ in range(args.steps):
            step()
        e1.record(st)
        torch.cuda.synchronize()
    barrier()
    J.jab_timing_enable(False)
    sites = J.jab_timing_read()
    ms = max_over_ranks(e0.elapsed_time(e1), dev)
    if J.jab_get_device_status() != 0:
        raise RuntimeError("device status set in the timed region")
    ms_step = ms / args.steps
    value = world * args.steps / (ms / 1e3)
    fwd_f, bwd_f = step_flops(wl)
    gpu_launches = sum(v[2] for v in sites.values())

    # ---- roofline of the dominant kernel (largest summed device time in the timed region)
    roofline = roofline_of(sites, scaled_work(wl, 1, args.steps), pk)
    dom = roofline["kernel"]
    traffic = None  # DRAM bytes per launch from an ncu capture, only while the kernel source is unchanged
    tfile = os.path.join(ROOT, "profiles", "traffic.json")
    if os.path.exists(tfile):
        import hashlib
        with open(tfile) as f:
            ent = json.load(f).get(f"{dom}@{wl.name}@B{wl.batch}xT{wl.seq_len}")
        if ent:
            csrc = os.path.join(ROOT, "paper_2609_34866_gb300", "csrc")
            same = all(hashlib.sha256(open(os.path.join(csrc, fn), "rb").read()).hexdigest()[:16] == h
                       for fn, h in ent.get("csrc_sha256_16", {}).items()
                       if os.path.exists(os.path.join(csrc, fn)))
            traffic = ent["bytes_per_launch"] if same else None
    roofline["traffic"] = traffic
    kernels = {k: {"ms_per_step": v[0] / args.steps, "launches_per_step": v[2] / args.steps}
               for k, v in sites.items()}

    # ---- forward-only rate (one candidate; converts X itself)
    def fwd_step():
        J.jab_loss_forward(desc, B, T, X, W, A, [bits], [scales], loss, ws)

    fwd_ms, _ = timed(J, fwd_step, args.steps, max(1, args.warmup), st, barrier, sites=False)
    fwd_ms = max_over_ranks(fwd_ms, dev)
    fwd_value = world * args.steps / (fwd_ms / 1e3)

    # ---- forward with both terms of Eq. 3 (MSE + 0.1 KL, one candidate; teacher projection once)
    qkv_ref = torch.empty((B, T, s.d_out), dtype=torch.float16, device=dev)
    J.jab_reference_projection(desc, B, T, X, W, qkv_ref, ws)

    def kl_step():
        J.jab_loss_forward_kl(desc, B, T, X, W, A, qkv_ref, [bits], [scales], 0.1, loss, ws)

    kl_ms, _ = timed(J, kl_step, args.steps, max(1, args.warmup), st, barrier, sites=False)
    kl_ms = max_over_ranks(kl_ms, dev)
    kl_f = fwd_f + work_of(wl)["attn_kl"][1]

    # ---- STE step on both terms of Eq. 3 (lambda_KL = 0.1): the scale gradient of MSE + 0.1 KL;
    # the teacher's projection and log-sum-exp are made once per calibration batch, like A_ref;
    # the call converts X itself
    lse_ref = torch.empty((B, s.n_q_heads, T), dtype=torch.float32, device=dev)
    J.jab_reference_forward(desc, B, T, X, W, A, ws, lse=lse_ref)

    def kl_bwd_step():
        J.jab_loss_backward_scales_kl(desc, B, T, X, W, A, qkv_ref, lse_ref, bits, scales, 0.0, 0.1,
                                      loss, grad, ws)
        if world > 1:
            combine_shards(loss, grad, B, B * world)

    n_klb = max(1, min(args.steps, 5))
    klb_ms, klb_sites = timed(J, kl_bwd_step, n_klb, max(1, min(args.warmup, 2)), st, barrier)
    klb_ms = max_over_ranks(klb_ms, dev)
    if J.jab_get_device_status() != 0:
        raise RuntimeError("device status set in the KL-term backward")
    J.jab_prepare_x(desc, B, T, X, ws)  # the headline's prepared X for what follows
    del qkv_ref, lse_ref
    klb_f = fwd_f + bwd_f + work_of(wl)["attn_kl"][1]

    # ---- Fisher-coupling probe (App. B): the loss and ||dL/dw_hat||^2 at 2 bits with round-to-
    # nearest (absmax) scales, one fwd + bwd per evaluation; reported beside the main metric
    s2 = scales_for(J, desc, wl, W, 2, dev, mode=0)
    sq = torch.empty(1, dtype=torch.float64, device=dev)

    def fisher_step():
        J.jab_loss_backward_weights(desc, B, T, X, W, A, 2, s2, loss, grad_sqnorm=sq, ws=ws)

    n_fis = max(1, min(args.steps, 3))
    fis_ms, _ = timed(J, fisher_step, n_fis, max(1, min(args.warmup, 2)), st, barrier, sites=False)
    fis_ms = max_over_ranks(fis_ms, dev)

    # ---- end to end through the C ABI with host buffers (pinned), copies inside the timed region.
    # Every step copies its own inputs (X, W, scales) host -> device and reads its result (loss,
    # scale gradient) back. The teacher output A(X; W) is not shipped: each step recomputes it on the
    # device from the X and W it received (jab_reference_forward, which also makes the fp16 copy of
    # X), then evaluates the loss and its gradient on that X (jab_loss_backward_scales_prepared).
    # Recomputing costs the teacher's projection and attention (~11 ms); copying the fp32 A_ref
    # (B T Hq d_h x 4 bytes, 4.29 GB here) would cost ~35-45 ms of a host link that tensor work
    # slows to ~100-125 GB/s. As in a fitting loop over changing batches, step i + 1's inputs are
    # copied on a second stream into the other of two device buffers while step i computes; the
    # first step's copy and every step's read-back are inside the timed region.
    e2e = None
    if not args.no_e2e:
        hosts = tuple(t.cpu().pin_memory() for t in (X, W, scales))
        dbuf = [tuple(torch.empty_like(t) for t in (X, W, scales)) for _ in range(2)]
        dA = torch.empty_like(A)  # the step's teacher output, made on the device
        hL = torch.empty(1, dtype=torch.float64).pin_memory()
        hG = torch.empty(grad.shape, dtype=torch.float32).pin_memory()
        cs = torch.cuda.Stream()
        copied = [torch.cuda.Event() for _ in range(2)]
        freed = [None, None]  # event after the last compute that read each buffer

        def copy_in(i):
            b = i % 2
            if freed[b] is not None:
                cs.wait_event(freed[b])
            with torch.cuda.stream(cs):
                for d_, h_ in zip(dbuf[b], hosts):
                    d_.copy_(h_, non_blocking=True)
                copied[b].record(cs)

        def compute(i):
            b = i % 2
            st.wait_event(copied[b])
            dX, dW, dS = dbuf[b]
            J.jab_reference_forward(desc, B, T, dX, dW, dA, ws, stream=st)
            J.jab_loss_backward_scales_prepared(desc, B, T, dX, dW, dA, bits, dS, 0.0, loss, grad,
                                                ws, stream=st)
            if world > 1:
                combine_shards(loss, grad, B, B * world)
            ev = torch.cuda.Event()
            ev.record(st)
            freed[b] = ev
            hL.copy_(loss, non_blocking=True)
            hG.copy_(grad, non_blocking=True)

        def e2e_run(n, start_event=None):
            if start_event is not None:
                cs.wait_event(start_event)
            copy_in(0)
            for i in range(n):
                if i + 1 < n:
                    copy_in(i + 1)
                compute(i)

        e2e_run(args.warmup)
        barrier()
        torch.cuda.synchronize()
        e0.record(st)
        e2e_run(args.steps, e0)
        e1.record(st)
        torch.cuda.synchronize()
        e2e_ms = max_over_ranks(e0.elapsed_time(e1), dev)
        if J.jab_get_device_status() != 0:
            raise RuntimeError("device status set in the end-to-end run")
        h2d = sum(t.numel() * t.element_size() for t in hosts)
        d2h = hL.numel() * 8 + hG.numel() * 4
        e2e = {"value": world * args.steps / (e2e_ms / 1e3), "unit": "evals/s",
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
               "ms_per_step": e2e_ms / args.steps,
               "teacher": "recomputed on the device every step from the copied X and W "
                          "(jab_reference_forward), not copied",
               "overlap": "step i+1's host-to-device copies overlap step i's compute (2 buffers)"}
        del hosts, dbuf, dA

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        # a bounded sample of ~10-20 s of oracle work: size it from one sequence's time
        dt1, _ = oracle_sample(wl, 1)
        k = max(1, min(wl.batch, int(np.ceil(12.0 / max(dt1, 1e-3)))))
        dt, sample = oracle_sample(wl, k) if k > 1 else (dt1, _)
        cpu = {"value": k / (dt * wl.batch), "unit": "evals/s", "cores": os.cpu_count(),
               "kind": "oracle", "sample": sample, "seconds": dt}

    return {
        "metric": METRIC, "value": value, "unit": "evals/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f16", "data": "synthetic",
        "config": {**config_of(wl), "x_f16": "converted once per calibration batch (jab_prepare_x): "
                                              "the scale fit's X is fixed across its steps",
                   "parallelism": ("single GPU" if world == 1 else
                                   f"sequence-sharded over {world} ranks: each rank a {B}-sequence "
                                   f"shard of a {B * world}-sequence batch, loss and scale gradient "
                                   "combined by one all-reduce per step")},
        **rates(fwd_f + bwd_f, ms_step, pk),
        "algorithmic_tflop_per_step": {"fwd": fwd_f / 1e12, "bwd": bwd_f / 1e12},
        "fwd_only": {"value": fwd_value, "unit": "evals/s", "ms_per_eval": fwd_ms / args.steps,
                     "achieved_tflops": fwd_f / (fwd_ms / args.steps / 1e3) / 1e12},
        "fwd_kl": {"value": world * args.steps / (kl_ms / 1e3), "unit": "evals/s",
                   "ms_per_eval": kl_ms / args.steps, "lambda_kl": 0.1,
                   "achieved_tflops": kl_f / (kl_ms / args.steps / 1e3) / 1e12},
        "fwd_bwd_kl": {"value": world * n_klb / (klb_ms / 1e3), "unit": "evals/s",
                       "ms_per_eval": klb_ms / n_klb, "lambda_kl": 0.1,
                       "achieved_tflops": klb_f / (klb_ms / n_klb / 1e3) / 1e12,
                       "note": "scale gradient of MSE + 0.1 KL (jab_loss_backward_scales_kl), "
                               "X converted by the call",
                       "kernels": {k: {"ms_per_step": v[0] / n_klb,
                                       "launches_per_step": v[2] / n_klb}
                                   for k, v in klb_sites.items()}},
        "fisher_probe": {"value": world * n_fis / (fis_ms / 1e3), "unit": "evals/s", "bits": 2,
                         "ms_per_eval": fis_ms / n_fis,
                         "achieved_tflops": (fwd_f + bwd_f) / (fis_ms / n_fis / 1e3) / 1e12},
        "roofline": roofline, "kernels": kernels, "cpu_baseline": cpu, "e2e": e2e,
        "gpu_launches": gpu_launches, "clocks": clk.summary(), "path": "tcgen05",
    }


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="mistral_block", choices=sorted(WORKLOADS))
    ap.add_argument("--batch", type=int, default=None,
                    help="override the workload's sequence count (smaller cases for profiling)")
    ap.add_argument("--seq-len", type=int, default=None, help="override the workload's sequence length")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-workloads", action="store_true",
                    help="skip the other workloads' throughput (reported under 'workloads')")
    args = ap.parse_args()
    wl = WORKLOADS[args.workload]
    if args.batch is not None or args.seq_len is not None:
        wl = wl.with_batch(args.batch or wl.batch, args.seq_len)
    if args.impl == "reference":
        return run_reference(args, wl)
    return run_ours(args, wl)


if __name__ == "__main__":
    sys.exit(main())
