#!/usr/bin/env python3
"""Throughput of the L_JAB hot path on GB300: candidate-loss evaluations per second.

One step = one forward L_JAB + STE/LSQ scale-gradient evaluation (jab_loss_backward_scales) of the
Mistral-7B-shaped attention block (d_model 4096, 32 query / 8 KV heads of 128, RoPE theta 1e4),
X = 128 sequences x 2048 tokens of Student-t(4) unit-variance activations, 3-bit groups of 128.
The teacher output A(X; W) is computed once before the timed region (it is shared by every
evaluation of the block, like the STE fitting loop's 200 steps). Reported beside it: the
forward-only rate (jab_loss_forward, one candidate) and the Fisher-coupling probe (loss and squared
STE weight-gradient norm at 2 bits, jab_loss_backward_weights).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference] [--workload NAME]

Under torchrun each rank evaluates its own seeded batch on its own GPU (independent units, no
collective on the data path): weak scaling, value = all ranks' evaluations / max rank time.
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

from paper_2609_34866_gb300.multi import dist_env, max_over_ranks  # noqa: E402
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
    """Algorithmic FLOPs / bytes per launch site (GEMM = 2MNK; causal attention counts the lower
    triangle including the diagonal; backward attention = 2.5x forward; no dX GEMM)."""
    s = wl.shape
    N, D, d = wl.batch * wl.seq_len, s.d_out, s.d_model
    attn = 4.0 * wl.batch * s.n_q_heads * s.head_dim * wl.seq_len * (wl.seq_len + 1) / 2
    return {
        "proj_gemm": ("flop", 2.0 * N * C * D * d),
        "attn_fwd": ("flop", attn * C),
        "attn_bwd": ("flop", 2.5 * attn),
        "wgrad_lsq": ("flop", 2.0 * N * D * d),
        "convert_x": ("byte", 4.0 * N * d),
        "transpose_x": ("byte", 4.0 * N * d),
        "quantize": ("byte", 4.0 * D * d),
    }


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
            "rope": s.use_rope, "bits": wl.bits[0], "group_size": wl.group_size,
            "x": f"{wl.x_dist}" + (f"(df={wl.x_df})" if wl.x_df else "") +
                 (f", {wl.outlier_frac:.1%} channels x{wl.outlier_factor:g}" if wl.outlier_frac else ""),
            "scale_init": wl.scale_init,
            "l2": "no flush: X (bf16) and A_ref (fp32) of every step are each larger than the 129 MB L2"}


# ------------------------------------------------------------------------------------ oracle timing
def oracle_sample(wl, seqs=1):
    """The float64 oracle's fwd+STE-bwd on `seqs` sequences of the workload (teacher precomputed,
    as in the GPU step). Returns (seconds, description)."""
    from oracle import jab_oracle as O
    s = wl.shape
    od = dict(d_model=s.d_model, n_q_heads=s.n_q_heads, n_kv_heads=s.n_kv_heads,
              head_dim=s.head_dim, group_size=wl.group_size, use_rope=s.use_rope,
              rope_theta=s.rope_theta, softmax_scale=0.0)
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
    s = wl.shape
    B, T = wl.batch, wl.seq_len
    desc = J.desc_from_shape(s, wl.group_size)
    X = make_x(wl, device=dev, seed=wl.seed + rank)
    W = make_block_weights(wl, device=dev)
    bits = wl.bits[0]
    scales = torch.empty((s.d_out, s.d_model // wl.group_size), dtype=torch.float32, device=dev)
    J.jab_init_scales(desc, bits, 1 if wl.scale_init == "minmse" else 0, W, scales)
    ws = J.Workspace(desc, B, T, 1, True, device=dev)
    A = torch.empty((B, T, s.n_q_heads * s.head_dim), dtype=torch.float32, device=dev)
    J.jab_reference_forward(desc, B, T, X, W, A, ws)
    loss = torch.empty(1, dtype=torch.float64, device=dev)
    grad = torch.empty_like(scales)
    st = torch.cuda.current_stream()

    def step():
        J.jab_loss_backward_scales(desc, B, T, X, W, A, bits, scales, 0.0, loss, grad, ws)

    def fwd_step():
        J.jab_loss_forward(desc, B, T, X, W, A, [bits], [scales], loss, ws)

    def barrier():
        if world > 1:
            torch.distributed.barrier()

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
    work = work_of(wl)
    dom = max(sites, key=lambda k: sites[k][0])
    dom_ms, dom_ranges, _ = sites[dom]
    per_launch_ms = dom_ms / max(1, dom_ranges)
    kind, amount = work.get(dom, ("flop", float("nan")))
    tc = os.environ.get("JAB_PATH", "tc") != "simple"
    if kind == "flop":
        achieved = amount / (per_launch_ms / 1e3) / 1e12
        if tc:
            bound, peak, unit = "tensor", pk["bf16_sus"], "TFLOP/s"
            peak_note = (f"{pk['source']} sustained bf16 dense (fp16 operands: same nominal rate)")
        else:
            peak = 152 * 128 * 2 * pk["sm_max_mhz"] * 1e6 / 1e12
            bound, unit = "alu", "TFLOP/s"
            peak_note = "FP32 FMA: 152 SMs x 128 lanes x 2 flop x max SM clock"
    else:
        achieved = amount / (per_launch_ms / 1e3) / 1e9
        bound, peak, unit = "hbm", pk["hbm"], "GB/s"
        peak_note = f"{pk['source']} HBM copy bandwidth"
    traffic = None  # DRAM bytes per launch from an ncu capture, only while the kernel source is unchanged
    tfile = os.path.join(ROOT, "profiles", "traffic.json")
    if os.path.exists(tfile):
        import hashlib
        with open(tfile) as f:
            ent = json.load(f).get(f"{dom}@{wl.name}@B{wl.batch}xT{wl.seq_len}@{'tc' if tc else 'simple'}")
        if ent:
            csrc = os.path.join(ROOT, "paper_2609_34866_gb300", "csrc")
            same = all(hashlib.sha256(open(os.path.join(csrc, fn), "rb").read()).hexdigest()[:16] == h
                       for fn, h in ent.get("csrc_sha256_16", {}).items()
                       if os.path.exists(os.path.join(csrc, fn)))
            traffic = ent["bytes_per_launch"] if same else None
    roofline = {"bound": bound, "achieved": achieved, "peak": peak, "unit": unit,
                "frac": achieved / peak, "traffic": traffic, "kernel": dom,
                "launch_ms": per_launch_ms, "peak_source": peak_note}
    kernels = {k: {"ms_per_step": v[0] / args.steps, "launches_per_step": v[2] / args.steps}
               for k, v in sites.items()}

    # ---- forward-only rate (one candidate)
    for _ in range(max(1, args.warmup)):
        fwd_step()
    barrier()
    torch.cuda.synchronize()
    e0.record(st)
    for _ in range(args.steps):
        fwd_step()
    e1.record(st)
    torch.cuda.synchronize()
    fwd_ms = max_over_ranks(e0.elapsed_time(e1), dev)
    fwd_value = world * args.steps / (fwd_ms / 1e3)

    # ---- Fisher-coupling probe (App. B): the loss and ||dL/dw_hat||^2 at 2 bits with round-to-
    # nearest (absmax) scales, one fwd + bwd per evaluation; reported beside the main metric
    s2 = torch.empty_like(scales)
    J.jab_init_scales(desc, 2, 0, W, s2)
    sq = torch.empty(1, dtype=torch.float64, device=dev)

    def fisher_step():
        J.jab_loss_backward_weights(desc, B, T, X, W, A, 2, s2, loss, grad_sqnorm=sq, ws=ws)

    n_fis = max(1, min(args.steps, 3))
    for _ in range(max(1, min(args.warmup, 2))):
        fisher_step()
    barrier()
    torch.cuda.synchronize()
    e0.record(st)
    for _ in range(n_fis):
        fisher_step()
    e1.record(st)
    torch.cuda.synchronize()
    fis_ms = max_over_ranks(e0.elapsed_time(e1), dev)
    if J.jab_get_device_status() != 0:
        raise RuntimeError("device status set during the Fisher-coupling probe")

    # ---- end to end through the C ABI with host buffers (pinned), copies inside the timed region.
    # Every step copies its own inputs (X, W, A_ref, scales) host -> device and reads its result
    # (loss, scale gradient) back. As in a fitting loop, step i + 1's inputs are copied on a second
    # stream into the other of two device buffers while step i computes; the first step's copy and
    # every step's read-back are inside the timed region.
    e2e = None
    if not args.no_e2e:
        hosts = tuple(t.cpu().pin_memory() for t in (X, W, A, scales))
        dbuf = [tuple(torch.empty_like(t) for t in (X, W, A, scales)) for _ in range(2)]
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
            dX, dW, dA, dS = dbuf[b]
            J.jab_loss_backward_scales(desc, B, T, dX, dW, dA, bits, dS, 0.0, loss, grad, ws, stream=st)
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
        h2d = sum(t.numel() * t.element_size() for t in hosts)
        d2h = hL.numel() * 8 + hG.numel() * 4
        e2e = {"value": world * args.steps / (e2e_ms / 1e3), "unit": "evals/s",
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
               "ms_per_step": e2e_ms / args.steps,
               "overlap": "step i+1's host-to-device copies overlap step i's compute (2 buffers)"}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        # a bounded sample of ~10-20 s of oracle work: size it from one sequence's time
        dt1, _ = oracle_sample(wl, 1)
        k = max(1, min(wl.batch, int(np.ceil(12.0 / max(dt1, 1e-3)))))
        dt, sample = oracle_sample(wl, k) if k > 1 else (dt1, _)
        cpu = {"value": k / (dt * wl.batch), "unit": "evals/s", "cores": os.cpu_count(),
               "kind": "oracle", "sample": sample, "seconds": dt}

    if world > 1:
        torch.distributed.destroy_process_group()
    if rank != 0:
        return 0
    tflops = (fwd_f + bwd_f) / (ms_step / 1e3) / 1e12
    line = {
        "metric": METRIC, "value": value, "unit": "evals/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f16", "data": "synthetic",
        "config": config_of(wl),
        "achieved_tflops": tflops,
        "frac_of_bf16_peak": {"burst": tflops / pk["bf16"], "sustained": tflops / pk["bf16_sus"],
                              "source": pk["source"]},
        "algorithmic_tflop_per_step": {"fwd": fwd_f / 1e12, "bwd": bwd_f / 1e12},
        "fwd_only": {"value": fwd_value, "unit": "evals/s", "ms_per_eval": fwd_ms / args.steps,
                     "achieved_tflops": fwd_f / (fwd_ms / args.steps / 1e3) / 1e12},
        "fisher_probe": {"value": world * n_fis / (fis_ms / 1e3), "unit": "evals/s", "bits": 2,
                         "ms_per_eval": fis_ms / n_fis,
                         "achieved_tflops": (fwd_f + bwd_f) / (fis_ms / n_fis / 1e3) / 1e12},
        "roofline": roofline, "kernels": kernels, "cpu_baseline": cpu, "e2e": e2e,
        "gpu_launches": gpu_launches, "clocks": clk.summary(),
        "path": "tcgen05" if tc else "cuda-core",
    }
    print(json.dumps(line), flush=True)
    return 0


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
    args = ap.parse_args()
    wl = WORKLOADS[args.workload]
    if args.batch is not None or args.seq_len is not None:
        wl = wl.with_batch(args.batch or wl.batch, args.seq_len)
    if args.impl == "reference":
        return run_reference(args, wl)
    return run_ours(args, wl)


if __name__ == "__main__":
    sys.exit(main())
