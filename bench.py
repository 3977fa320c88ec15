#!/usr/bin/env python
"""Benchmark of one NormPre optimizer step over a synthetic model parameter set.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--config NAME]

A step is the whole hot path (momentum, relaxed tangent, diagonal-Gram
normalization, spectral preconditioning, RMS-matched weight update with decay)
over every matrix of the parameter set.  Default workload: the GPT-2 Small
hidden matrices under NormPre-G (48 matrices, 84.9 M parameters, bf16
gradients, fp32 weights and momentum, 5 Newton-Schulz iterations).

Prints one JSON line: `value` is the device-timed ms per parameter-set step
(inputs resident in HBM), `e2e` the same step through the C ABI on pinned host
buffers with the copies inside the timed region, `roofline` the dominant
kernel class (the Newton-Schulz GEMMs for NormPre-G) against the measured
peak, `cpu_baseline` the fp64 oracle on the host cores for a bounded sample.
`--impl reference` times the oracle itself on the same workload.
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

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from synth import inputs as S  # noqa: E402

METRIC = "NormPre step ms per model param set; NS TFLOP/s & normalize GB/s vs peak"
DEFAULT_CONFIG = "gpt2_small_G"
LR = 0.02
# Traffic of one launch of the dominant kernel class from an ncu capture
# (dram__bytes_read.sum + dram__bytes_write.sum), per workload; None until a
# capture of the current kernel exists (profiles/ keeps the summaries).
FP32_FMA_TFLOPS = 152 * 128 * 2 * 2.07e9 / 1e12   # 80.5 TFLOP/s, for the ALU-bound k_gamma
L2_BYTES = 129e6                                    # GB300 L2

NCU_TRAFFIC_PER_LAUNCH = {
    "gpt2_small_G": 208.1e6,   # mean of 15 launches: Gram, poly and update of five NS iterations
    "gpt2_small_L": 108.0e6,   # mean of six k_contract_tc launches (both operand orientations)
}


# ---------------------------------------------------------------------------
# helpers
# ---------------------------------------------------------------------------
def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d.get("hbm_gbs"), d.get("bf16_tflops"), d.get("bf16_tflops_sustained"), "measured"
    return 6800.0, 1900.0, 1700.0, "fallback"


def ns_flops(cfg: S.ParamSetConfig, steps: int) -> float:
    """Algorithmic Newton-Schulz flops of one step: per iteration and matrix
    2 s^2 big (Gram) + 2 s^3 (A A) + 2 s^2 big (B X), s = min(m, n)."""
    tot = 0.0
    for m in cfg.matrices:
        s, big = min(m.rows, m.cols), max(m.rows, m.cols)
        tot += steps * (4.0 * s * s * big + 2.0 * s ** 3)
    return tot


def ns_executed_flops(cfg: S.ParamSetConfig, steps: int) -> float:
    """Flops the tensor-core path executes in one step.  Dimensions are padded
    (the short side s to 128, the long side to 256), the Gram and polynomial
    products compute only the 128 x BN tiles that reach the diagonal (BN = 256
    when the padded s is a multiple of 256, else 128) and mirror the rest."""
    def up(x, m):
        return (x + m - 1) // m * m
    tot = 0.0
    for m in cfg.matrices:
        s, big = min(m.rows, m.cols), max(m.rows, m.cols)
        sp, bp = up(s, 128), up(big, 256)
        bn = 256 if sp % 256 == 0 else 128
        tiles_m, tiles_n, rr = sp // 128, sp // bn, bn // 128
        sym_tiles = sum(min(rr * (c + 1), tiles_m) for c in range(tiles_n))
        gram = 2.0 * sym_tiles * 128 * bn * bp
        poly = 2.0 * sym_tiles * 128 * bn * sp
        update = 2.0 * sp * bp * sp
        tot += steps * (gram + poly + update)
    return tot


def bytes_per_elt(cfg: S.ParamSetConfig, variant: str):
    g = 2 if cfg.g_dtype == "bf16" else 4
    w = 2 if cfg.w_dtype == "bf16" else 4
    psi = 2 if variant == "G" else 4        # bf16 Newton-Schulz input, fp32 for the L variants
    normalize = g + 4 + 4 + w + psi          # read G, M, W; write M, Psi
    apply = psi + 2 * w                      # read T (or Psi), read/write W
    return normalize, apply


class ClockSampler:
    """Samples nvidia-smi SM clocks and throttle reasons in the background."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index=None):
        self.rows = []
        self.proc = None
        self.gpu_index = gpu_index

    def start(self):
        cmd = ["nvidia-smi", "--query-gpu=" + self.FIELDS, "--format=csv,noheader,nounits", "-lms", "25"]
        if self.gpu_index is not None:
            cmd[1:1] = ["-i", str(self.gpu_index)]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) >= 9:
                self.rows.append(parts)

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.thread.join(timeout=2)

    def summary(self):
        if not self.rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        def num(x):
            try:
                return float(x)
            except ValueError:
                return None
        sm = [num(r[1]) for r in self.rows if num(r[1]) is not None]
        smax = [num(r[2]) for r in self.rows if num(r[2]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in self.rows for i in range(4) if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "reasons": reasons, "samples": len(self.rows)}


def max_over_ranks(x: float, world: int, device: str) -> float:
    """The largest value over the ranks of the process group (the job's time
    is its slowest rank's); x itself when there is one rank."""
    if world <= 1:
        return x
    import torch
    import torch.distributed as dist
    tt = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(tt, op=dist.ReduceOp.MAX)
    return float(tt.item())


def oracle_sample(cfg: S.ParamSetConfig, variant: str, seconds_budget: float = 20.0):
    """Times the fp64 oracle on a bounded sample of the workload (one layer's
    matrices of each distinct shape) and scales to the whole parameter set by
    matrix counts.  Returns (ms per parameter set, description, cores)."""
    import oracle as O
    from synth.inputs import make_matrix
    shapes = {}
    for i, m in enumerate(cfg.matrices):
        shapes.setdefault((m.rows, m.cols), []).append(i)
    oc = O.OracleConfig(variant=variant, rank=cfg.rank, oversample=0 if variant == "L_exact" else cfg.oversample,
                        power_iters=cfg.power_iters, seed=1234)
    total_ms = 0.0
    sampled = []
    for shp, idx in shapes.items():
        mats = make_matrix(cfg, idx[0])
        t0 = time.perf_counter()
        O.normpre_step(mats["W"], mats["G"], mats["M"], 0, LR, oc, matrix_id=idx[0])
        dt = (time.perf_counter() - t0) * 1e3
        total_ms += dt * len(idx)
        sampled.append("%dx%d" % shp)
    try:
        from threadpoolctl import threadpool_info
        cores = max([d.get("num_threads", 1) for d in threadpool_info()] + [1])
    except Exception:
        cores = os.cpu_count() or 1
    desc = ("oracle (numpy fp64) on one matrix of each distinct shape (%s), scaled by the matrix "
            "count of each shape to the %d-matrix set" % (", ".join(sampled), cfg.n_mats))
    return total_ms, desc, cores


# ---------------------------------------------------------------------------
# reference arm: the oracle as it stands, on the host cores
# ---------------------------------------------------------------------------
def run_reference(args, cfg, variant, rank, world):
    if rank != 0:
        return
    for _ in range(args.warmup):
        oracle_sample(cfg, variant)
    times = []
    desc, cores = "", 1
    for _ in range(args.steps):
        ms, desc, cores = oracle_sample(cfg, variant)
        times.append(ms)
    v = float(np.mean(times))
    line = {"metric": METRIC, "value": v, "unit": "ms", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": v, "higher_is_better": False, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "impl": "reference",
            "config": {"workload": cfg.name, "variant": variant, "n_mats": cfg.n_mats,
                       "elements": cfg.elements},
            "cpu_baseline": {"value": v, "unit": "ms", "cores": cores, "kind": "oracle", "sample": desc},
            "e2e": {"value": v, "unit": "ms", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------
# our arm
# ---------------------------------------------------------------------------
def run_ours(args, cfg, variant, rank, world):
    import torch
    import torch.distributed as dist

    from paper_2609_36692_gb300 import build as B
    B.build()
    from paper_2609_36692_gb300 import normpre as C
    from paper_2609_36692_gb300.optim import NormPre

    dev = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream()

    mats = S.make_param_set(cfg, workers=min(16, os.cpu_count() or 1))
    tdt = {"f32": torch.float32, "bf16": torch.bfloat16}
    W = [torch.from_numpy(m["W"]).to(tdt[cfg.w_dtype]).cuda() for m in mats]
    G = [torch.from_numpy(m["G"]).to(tdt[cfg.g_dtype]).cuda() for m in mats]
    M = [torch.from_numpy(m["M"]).cuda() for m in mats]
    prec = C.NORMPRE_PREC_BF16 if variant == "G" else C.NORMPRE_PREC_F32
    vcode = {"G": C.NORMPRE_G, "L": C.NORMPRE_L, "L_exact": C.NORMPRE_L_EXACT}[variant]
    opt = NormPre([(m.rows, m.cols) for m in cfg.matrices], [cfg.w_dtype] * cfg.n_mats,
                  [cfg.g_dtype] * cfg.n_mats, variant=vcode,
                  precision=prec, rank=cfg.rank, oversample=cfg.oversample,
                  power_iters=cfg.power_iters, ns_steps=cfg.ns_steps, seed=1234)
    h = opt.handle

    def barrier():
        if world > 1:
            dist.barrier()

    sampler = ClockSampler(gpu_index=dev)
    t = 0
    for _ in range(max(args.warmup, 3)):
        opt.step(t, LR, W, G, M)
        t += 1
    torch.cuda.synchronize()
    opt.status()
    C.normpre_profile_read(h)           # reset launch counters

    # ---- timed region: K steps, inputs resident in HBM (> L2 in total) ----
    sampler.start()
    time.sleep(0.1)                     # let the sampler's first query land
    barrier()
    torch.cuda.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(args.steps):
        opt.step(t, LR, W, G, M)
        t += 1
    ev1.record(stream)
    torch.cuda.synchronize()
    barrier()
    ms_total = ev0.elapsed_time(ev1)
    sampler.stop()
    counts = C.normpre_profile_read(h)
    launches = int(sum(c for _, c in counts.values()))
    opt.status()
    clocks = sampler.summary()
    clocks["source"] = "timed region"
    if clocks["samples"] < 3:
        # the timed region was too short to sample: keep the same load running
        # (untimed) for ~1.5 s and record the clocks it sees
        soak = ClockSampler(gpu_index=dev)
        soak.start()
        t_end = time.perf_counter() + 1.5
        while time.perf_counter() < t_end:
            for _ in range(10):
                opt.step(t, LR, W, G, M)
                t += 1
            torch.cuda.synchronize()
        soak.stop()
        clocks = soak.summary()
        clocks["source"] = "1.5 s soak of the same step right after the timed region (too short to sample)"
    ms_step = ms_total / args.steps
    ms_step = max_over_ranks(ms_step, world, "cuda")

    # ---- per-step distribution: a separate pass with one event pair per step
    # (row- and column-active steps alternate, so p10 and p90 tell them apart) ----
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(args.steps)]
    for e_a, e_b in evs:
        e_a.record(stream)
        opt.step(t, LR, W, G, M)
        t += 1
        e_b.record(stream)
    torch.cuda.synchronize()
    per_step = [e_a.elapsed_time(e_b) for e_a, e_b in evs]
    p10, p50, p90 = (float(v) for v in np.percentile(per_step, [10, 50, 90]))
    step_dist = {"p10": p10, "p50": p50, "p90": p90, "steps": len(per_step),
                 "source": "untimed pass after the timed region, one event pair per step"}

    # ---- per-kernel-class time of the same workload (events on the launch stream) ----
    C.normpre_profile(h, True)
    for _ in range(args.steps):
        opt.step(t, LR, W, G, M)
        t += 1
    torch.cuda.synchronize()
    prof = C.normpre_profile_read(h)
    C.normpre_profile(h, False)

    hbm, bf16_burst, bf16_sust, peak_src = measured_peaks()
    n_el = cfg.elements
    b_norm, b_apply = bytes_per_elt(cfg, variant)
    norm_ms = prof["normalize"][0] / args.steps
    phases = {k: {"ms_per_step": v[0] / args.steps, "launches_per_step": v[1] / args.steps}
              for k, v in prof.items() if v[1] > 0}
    if variant == "G":
        fl = ns_flops(cfg, cfg.ns_steps)
        fl_exec = ns_executed_flops(cfg, cfg.ns_steps)
        ns_ms = sum(prof[k][0] for k in ("ns_gram", "ns_poly", "ns_update")) / args.steps
        ns_launches = sum(prof[k][1] for k in ("ns_gram", "ns_poly", "ns_update")) / args.steps
        achieved = fl / (ns_ms * 1e-3) / 1e12
        # a step that ran into the power cap is held to the sustained matmul rate
        capped = "sw_power_cap" in clocks.get("reasons", [])
        peak = bf16_sust if capped else bf16_burst
        roof = {"bound": "tensor", "kernel": "k_ns_gemm_tc (Newton-Schulz Gram / poly / update)",
                "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                "frac": achieved / peak,
                "peak_source": "%s bf16 %s" % (peak_src, "sustained (sw_power_cap seen in the timed region)"
                                                if capped else "burst"),
                "flops_per_launch": fl / ns_launches, "ms_per_launch": ns_ms / ns_launches,
                "flops_note": "nominal dense flops (full Gram); the kernel computes only the "
                              "tiles on or above the diagonal of the two symmetric products",
                "executed_flops_per_launch": fl_exec / ns_launches,
                "achieved_executed": fl_exec / (ns_ms * 1e-3) / 1e12,
                "frac_executed": fl_exec / (ns_ms * 1e-3) / 1e12 / peak,
                "traffic": NCU_TRAFFIC_PER_LAUNCH.get(cfg.name)}
    elif variant == "L_exact":
        # k_gamma: Gamma = Psi_a Psi_a^T on the fp32 FMA pipes (both triangles,
        # 2 m_a^2 n_a flops per matrix); the dense eigensolver is a library call
        gam_ms = prof["gamma"][0] / args.steps
        gam_launches = prof["gamma"][1] / args.steps
        k_even = sum(2.0 * m.rows * m.rows * m.cols for m in cfg.matrices)
        k_odd = sum(2.0 * m.cols * m.cols * m.rows for m in cfg.matrices)
        fl = (k_even + k_odd) / 2.0          # row- and column-active steps alternate
        achieved = fl / (gam_ms * 1e-3) / 1e12
        fp32_peak = FP32_FMA_TFLOPS
        roof = {"bound": "alu", "kernel": "k_gamma (Gamma = Psi_a Psi_a^T, fp32 FMA)",
                "achieved": achieved, "peak": fp32_peak, "unit": "TFLOP/s", "frac": achieved / fp32_peak,
                "peak_source": "nominal fp32 FMA rate: 152 SMs x 128 lanes x 2 flops x 2.07 GHz",
                "flops_per_launch": fl / gam_launches, "ms_per_launch": gam_ms / gam_launches,
                "syevd_ms_per_step": prof["syevd"][0] / args.steps,
                "traffic": None}
    else:
        con_ms = prof["contract"][0] / args.steps
        con_launches = prof["contract"][1] / args.steps
        # each contraction streams the fp32 Psi of its group once: Y0 = Psi Omega,
        # Psi^T Y and Psi Z per power iteration, B = Q^T Psi
        nbytes = n_el * 4.0 * (2 + 2 * cfg.power_iters)
        achieved = nbytes / (con_ms * 1e-3) / 1e9
        roof = {"bound": "hbm", "kernel": "k_contract_tc (sketch contractions of Psi, tcgen05 TF32 split)",
                "achieved": achieved, "peak": hbm, "unit": "GB/s", "frac": achieved / hbm,
                "peak_source": "%s HBM copy bandwidth" % peak_src,
                "bytes_per_launch": nbytes / con_launches, "ms_per_launch": con_ms / con_launches,
                "traffic": NCU_TRAFFIC_PER_LAUNCH.get(cfg.name)}
    norm_gbs = n_el * b_norm / (norm_ms * 1e-3) / 1e9 if norm_ms > 0 else None

    # ---- end to end through the C ABI on pinned host buffers ----
    Wh = [torch.from_numpy(m["W"]).to(tdt[cfg.w_dtype]).pin_memory() for m in mats]
    Gh = [torch.from_numpy(m["G"]).to(tdt[cfg.g_dtype]).pin_memory() for m in mats]
    Mh = [torch.from_numpy(m["M"]).pin_memory() for m in mats]
    h2d = sum(x.numel() * x.element_size() for x in Wh + Gh + Mh)
    d2h = sum(x.numel() * x.element_size() for x in Wh + Mh)
    opt.step_host(t, LR, Wh, Gh, Mh)
    t += 1
    barrier()
    n_e2e = max(3, min(args.steps, 20))
    t0 = time.perf_counter()
    for _ in range(n_e2e):
        opt.step_host(t, LR, Wh, Gh, Mh)
        t += 1
    e2e_ms = (time.perf_counter() - t0) * 1e3 / n_e2e
    e2e_ms = max_over_ranks(e2e_ms, world, "cuda")

    # ---- the paper's comparison optimizer (Muon) on the same workload and kernels ----
    muon = None
    if not args.no_muon:
        opt_m = NormPre([(m.rows, m.cols) for m in cfg.matrices], [cfg.w_dtype] * cfg.n_mats,
                        [cfg.g_dtype] * cfg.n_mats, variant=C.NORMPRE_MUON, precision=C.NORMPRE_PREC_BF16,
                        ns_steps=cfg.ns_steps)
        for _ in range(max(args.warmup, 3)):
            opt_m.step(t, LR, W, G, M)
            t += 1
        torch.cuda.synchronize()
        barrier()
        ev0.record(stream)
        for _ in range(args.steps):
            opt_m.step(t, LR, W, G, M)
            t += 1
        ev1.record(stream)
        torch.cuda.synchronize()
        ms_muon = ev0.elapsed_time(ev1) / args.steps
        opt_m.status()
        opt_m.close()
        ms_muon = max_over_ranks(ms_muon, world, "cuda")
        muon = {"ms_per_step": ms_muon, "normpre_vs_muon": ms_step / ms_muon - 1.0,
                "paper_a100_context": "optimizer latency vs Muon on A100: NormPre-G +5.76 % / +4.37 % / +6.77 %, "
                                      "NormPre-L -38.12 % / -67.00 % / -57.16 % (GPT-2 Small / LLaMA-1.3B / "
                                      "Qwen3-1.7B, whole optimizer step incl. AdamW on the other parameters)"}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        ms_cpu, desc, cores = oracle_sample(cfg, variant)
        cpu = {"value": ms_cpu, "unit": "ms", "cores": cores, "kind": "oracle", "sample": desc}

    if rank == 0:
        line = {"metric": METRIC, "value": ms_step / world, "unit": "ms", "n_gpus": world,
                "steps": args.steps, "warmup": max(args.warmup, 3), "ms_per_step": ms_step,
                "higher_is_better": False, "scaling": "weak", "vs_baseline": None,
                "dtype": "bf16" if variant == "G" else "f32", "data": "synthetic",
                "config": {"workload": cfg.name, "variant": variant, "n_mats": cfg.n_mats,
                           "elements": n_el, "ns_steps": cfg.ns_steps if variant == "G" else None,
                           "rank": cfg.rank if variant in ("L", "L_exact") else None,
                           "l2": ("inputs larger than L2 (W, G, M = %.0f MB)" if h2d > L2_BYTES else
                                  "inputs within L2 (W, G, M = %.0f MB): a latency-scale workload, "
                                  "not flushed between steps") % (h2d / 1e6),
                           "parallelism": "replicas" if world > 1 else "single"},
                "e2e": {"value": e2e_ms / world, "unit": "ms", "h2d_bytes_per_step": h2d,
                        "d2h_bytes_per_step": d2h},
                "gpu_launches": launches,
                "step_ms": step_dist,
                "roofline": roof,
                "normalize": {"achieved": norm_gbs, "peak": hbm, "unit": "GB/s",
                              "frac": (norm_gbs / hbm) if norm_gbs else None,
                              "bytes_per_element": b_norm},
                "phases": phases,
                "muon": muon,
                "cpu_baseline": cpu,
                "clocks": clocks}
        print(json.dumps(line), flush=True)
    opt.close()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", default=DEFAULT_CONFIG, choices=sorted(S.CONFIGS))
    ap.add_argument("--variant", default=None, choices=[None, "G", "L", "L_exact"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-muon", action="store_true", help="skip timing the Muon comparison step")
    args = ap.parse_args()
    cfg = S.CONFIGS[args.config]
    variant = args.variant or cfg.variants[0]
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        if args.impl == "ours":
            import torch
            torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
        dist.init_process_group("nccl" if args.impl == "ours" else "gloo")
    if args.impl == "reference":
        run_reference(args, cfg, variant, rank, world)
    else:
        run_ours(args, cfg, variant, rank, world)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
