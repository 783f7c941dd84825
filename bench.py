#!/usr/bin/env python
"""Benchmark of BAG's cached DiT sampling path on one GB300 (or N independent replicas).

A "step" of this benchmark is one whole sample: T = 50 flow-matching steps of the
FLUX.1-dev-shaped MMDiT (19 double-stream + 38 single-stream blocks, hidden 3072,
4096 image + 512 text tokens) under budget B, i.e. exactly B full network evaluations
and T - B cached-residual steps, with the gate deciding on the device.

Printed (one JSON line, rank 0): s/sample (lower is better) as whole-job throughput,
an end-to-end figure through the host-buffer entry point, the roofline of the dominant
kernel class (tensor-core GEMM) from a profiled sample, and the fp64 oracle timed on
the host cores on a bounded sample of the same workload.

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--budget B]
                       [--impl ours|reference] [--config flux]
Under torchrun (N > 1) every rank runs its own replica (no collective on the data
path); the barrier + max-over-ranks timing follows the benchmark contract.
"""

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "s/sample at budget B (FLUX-shaped 1024², T=50); DiT-block TFLOPS vs bf16 peak"
# paper's number for the same budget on the FLUX 1024^2 50-step sampler (Tab. 1, BAG
# rows), measured on one RTX 4090 for the whole pipeline: context, not a target
PAPER_S_PER_SAMPLE = {20: 12.81, 13: 8.48, 9: 5.99}


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return p, "measured"
    except OSError:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


# ---------------------------------------------------------------------------
# clocks sampled during the timed region
# ---------------------------------------------------------------------------
class Clocks:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.path = tempfile.mktemp(prefix="bag_clocks_", suffix=".csv")
        self.gpu = gpu_index
        self.proc = None

    def start(self):
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"], stdout=self.f,
                stderr=subprocess.DEVNULL)
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
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    smax.append(float(parts[2]))
                except ValueError:
                    continue
                for n, v in zip(names, parts[5:9]):
                    if v.lower().startswith("active"):
                        reasons.add(n)
        os.unlink(self.path)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None, "reasons": sorted(reasons),
                "samples": len(sm)}


# ---------------------------------------------------------------------------
# fp64 oracle on the host cores (CPU baseline and the reference arm)
# ---------------------------------------------------------------------------
def cpu_worker(cfg_name, reps, warm):
    """Time the oracle's forward of one block of each kind the stack has (double-stream,
    single-stream, or Wan) at full width and full token count; print per-rep seconds."""
    import numpy as np

    from oracle import bag_oracle as O
    from paper_2608_09231_gb300 import configs, synth

    cfg = configs.get_config(cfg_name)
    types = synth.block_types(cfg)
    pick = sorted({types.index(t) for t in set(types)})
    W = O.to64(synth.make_weights(cfg, blocks=pick))
    G = W["global"]
    inp = synth.make_inputs(cfg)
    H = cfg["heads"]
    vec = O.conditioning(cfg, G, 1.0, inp["pooled"].astype(np.float64))
    img = O.patch_embed(G, inp["x"].astype(np.float64))
    txt = inp["txt"].astype(np.float64)
    ang = O.rope_angles(O.token_positions(cfg), cfg["rope_axes"])
    out = []
    for r in range(warm + reps):
        rec = {"double_s": 0.0, "single_s": 0.0, "wan_s": 0.0}
        for b in pick:
            blk = W["blocks"][b]
            mod = O.block_modulation(cfg, G, blk, vec)
            t0 = time.perf_counter()
            if blk["type"] == "double":
                O.double_block(img, txt, mod[0], mod[1], blk, ang, H)
            elif blk["type"] == "single":
                O.single_block(np.concatenate([txt, img], axis=0), mod, blk, ang, H)
            else:
                O.wan_block(img, txt, mod, blk, ang, H)
            rec[blk["type"] + "_s"] = time.perf_counter() - t0
        if r >= warm:
            out.append(rec)
    print(json.dumps({"reps": out, "threads": os.cpu_count()}))


def run_cpu_oracle(cfg_name, reps, warm):
    env = dict(os.environ)
    n = str(os.cpu_count() or 1)
    for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        env[k] = n
    env["CUDA_VISIBLE_DEVICES"] = ""
    r = subprocess.run([sys.executable, os.path.abspath(__file__), "--cpu-worker", cfg_name,
                        str(reps), str(warm)], capture_output=True, text=True, env=env,
                       cwd=ROOT)
    if r.returncode != 0:
        raise RuntimeError("oracle worker failed: " + r.stderr[-2000:])
    return json.loads(r.stdout.strip().splitlines()[-1])


def oracle_s_per_sample(cfg, B, rep):
    """Extrapolate one oracle sample: B full forwards of the whole stack (of both
    branches under classifier-free guidance)."""
    branches = 1 if cfg.get("guidance") is None else 2
    return branches * B * (cfg["n_double"] * rep["double_s"] + cfg["n_single"] * rep["single_s"]
                           + cfg["n_wan"] * rep["wan_s"])


# ---------------------------------------------------------------------------
KERNEL_NAMES = {"gemm": "gemm_tc_kernel", "attention": "attn_tc_kernel",
                "norm": "ln_mod_kernel", "signal": "ln_mod_kernel (signal)",
                "gate": "gate_kernel", "cache": "cache_refresh/reuse_kernel"}
KERNEL_SOURCES = {"gemm_tc_kernel": ["gemm.cu", "epilogue.cuh", "common.cuh"],
                  "gemm_pair_kernel": ["gemm.cu", "epilogue.cuh", "common.cuh"],
                  "attn_tc_kernel": ["attn_tc.cu", "common.cuh"]}


def source_sha1(kernel):
    h = hashlib.sha1()
    for f in KERNEL_SOURCES.get(kernel, []):
        with open(os.path.join(ROOT, "paper_2608_09231_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def measured_traffic(kernel, shape):
    """DRAM bytes per launch from the committed ncu summary, if it was taken on the
    current source of that kernel (else None)."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        entries = json.load(f).get("entries", [])
    for e in entries:
        if (e.get("kernel") == kernel and list(e.get("shape", [])) == list(shape)
                and e.get("source_sha1") == source_sha1(kernel)):
            return e.get("dram_bytes_per_launch")
    return None


def dominant_roofline(recs, peaks, peak_src, cfg_name, f32=False):
    """Roofline of the (kernel, shape) group that takes the most event time.  fp32
    configurations run on the CUDA cores; their bound is the fp32 FMA rate."""
    groups = {}
    for r in recs:
        key = (r["kind"], r["m"], r["n"], r["k"], r.get("variant", 0))
        g = groups.setdefault(key, {"launches": 0, "ms": 0.0, "flops": 0.0, "bytes": 0.0})
        g["launches"] += 1
        g["ms"] += r["ms"]
        g["flops"] += r["flops"]
        g["bytes"] += r["bytes"]
    kind, m, n, k, variant = max(groups, key=lambda q: groups[q]["ms"])
    g = groups[(kind, m, n, k, variant)]
    name = KERNEL_NAMES[kind]
    if kind == "gemm" and variant == 1:
        name = "gemm_pair_kernel"
    if f32 and kind in ("gemm", "attention"):
        name = {"gemm": "gemm_simt_kernel", "attention": "attn_simt_kernel"}[kind]
    avg_ms = g["ms"] / g["launches"]
    total = sum(v["ms"] for v in groups.values())
    shape = [m, n, k]
    if g["flops"] > 0 and f32:
        # fp32 FMA peak from the unit counts and clock: 152 SMs x 128 FMA/clk x 2 flop x
        # sm_max_mhz (the fp32 configuration is a parity check, not a throughput target)
        per = g["flops"] / g["launches"]
        ach = per / (avg_ms * 1e-3) / 1e12
        peak = 152 * 128 * 2 * peaks.get("sm_max_mhz", 2070.0) * 1e6 / 1e12
        return {"bound": "alu", "kernel": name, "shape": shape, "achieved": ach, "peak": peak,
                "unit": "TFLOP/s", "frac": ach / peak, "traffic": None,
                "peak_source": "fp32 FMA: 152 SMs x 128 lanes x 2 flop x max SM clock",
                "launches": g["launches"], "avg_launch_ms": avg_ms, "flops_per_launch": per,
                "share_of_profiled_time": g["ms"] / total}
    if g["flops"] > 0:
        per = g["flops"] / g["launches"]
        ach = per / (avg_ms * 1e-3) / 1e12
        peak = peaks.get("bf16_tflops_sustained", 1700.0)
        return {"bound": "tensor", "kernel": name, "shape": shape, "achieved": ach, "peak": peak,
                "unit": "TFLOP/s", "frac": ach / peak, "traffic": measured_traffic(name, shape),
                "peak_source": f"{peak_src} bf16 sustained (kernel timed inside the step)",
                "launches": g["launches"], "avg_launch_ms": avg_ms, "flops_per_launch": per,
                "share_of_profiled_time": g["ms"] / total}
    per = g["bytes"] / g["launches"]
    ach = per / (avg_ms * 1e-3) / 1e9
    peak = peaks.get("hbm_gbs", 6800.0)
    return {"bound": "hbm", "kernel": name, "shape": shape, "achieved": ach, "peak": peak,
            "unit": "GB/s", "frac": ach / peak, "traffic": measured_traffic(name, shape),
            "peak_source": f"{peak_src} HBM copy", "launches": g["launches"],
            "avg_launch_ms": avg_ms, "bytes_per_launch": per,
            "share_of_profiled_time": g["ms"] / total}


BLOCK_WORKLOADS = {
    "flux": ("flux_block", {}, "FLUX-shaped single-stream block, 4096 img + 512 txt tokens, "
             "d 3072, 24x128 heads, MLP 12288, bf16"),
    "qwen": ("qwen", {"n_double": 1}, "Qwen-Image-shaped double-stream block, 6889 img + 256 "
             "txt tokens, d 3072, 24x128 heads, MLP 12288, bf16"),
    "wan": ("wan", {"n_wan": 1}, "Wan2.1-14B-shaped block (self-attention over 32760 tokens, "
            "cross-attention to 512, FFN 13824), d 5120, 40x128 heads, bf16"),
}


def block_flops(cfg):
    """Algorithmic flops of one block forward: its projections and attention."""
    d, F, ni, nx = cfg["hidden"], cfg["mlp"], cfg["n_img"], cfg["n_txt"]
    if cfg["kind"] == "wan":
        return (2.0 * ni * d * 3 * d + 4.0 * ni * ni * d + 2.0 * ni * d * d          # self-attn
                + 2.0 * ni * d * d + 2.0 * nx * d * 2 * d + 4.0 * ni * nx * d      # cross-attn
                + 2.0 * ni * d * d + 4.0 * ni * d * F)                             # out, FFN
    N = ni + nx
    if cfg["n_double"] > 0:
        return 2.0 * N * d * 3 * d + 4.0 * N * N * d + 2.0 * N * d * d + 4.0 * N * d * F
    return 2.0 * N * d * (3 * d + F) + 2.0 * N * (d + F) * d + 4.0 * N * N * d


def block_mode(args):
    """One block forward at a benchmark model's full width and token count (--config
    flux: a FLUX single-stream block; qwen: a Qwen-Image double-stream block; wan: a
    Wan2.1-14B block) and the skip-path kernel: the per-block throughput of the stack
    and the cost of a reused step.  Also the target of the ncu captures."""
    import numpy as np
    import torch

    from paper_2608_09231_gb300 import bag, configs, synth

    name, over, workload = BLOCK_WORKLOADS[args.config]
    cfg = configs.get_config(name, qk_norm=args.qk_norm, **over)
    d = cfg["hidden"]
    N = cfg["n_img"] + (0 if cfg["kind"] == "wan" else cfg["n_txt"])
    ctx = bag.create(cfg, T=cfg["T"], B=1)
    stream = torch.cuda.current_stream()
    ctx.set_stream(stream.cuda_stream)
    inp = synth.make_inputs(cfg)
    txt = torch.from_numpy(inp["txt"]).cuda().to(torch.bfloat16)
    pooled = torch.from_numpy(inp["pooled"]).cuda()
    ctx.prepare(txt, pooled)
    h0 = torch.from_numpy(synth.normal(cfg["weight_seed"], 900, N * d, 1.0)).cuda().reshape(N, d)
    h = h0.clone()
    for _ in range(args.warmup):
        ctx.forward_block(0, 0, h)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(True), torch.cuda.Event(True)
    e0.record(stream)
    for _ in range(args.steps):
        ctx.forward_block(0, 0, h)
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / args.steps
    flops = block_flops(cfg)
    # skip path: h_out = h_in + R over the image stream
    n = cfg["n_img"] * d
    hin = h0[:cfg["n_img"]].contiguous()
    R = torch.from_numpy(synth.normal(cfg["weight_seed"], 901, n, 0.3)).cuda()
    out = torch.empty_like(hin)
    for _ in range(3):
        ctx.residual_add(out, hin, R, n)
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(20):
        ctx.residual_add(out, hin, R, n)
    e1.record(stream)
    torch.cuda.synchronize()
    ms_skip = e0.elapsed_time(e1) / 20
    peaks, src = _peaks()
    tf = flops / (ms * 1e-3) / 1e12
    gbs = 12.0 * n / (ms_skip * 1e-3) / 1e9
    print(json.dumps({"mode": "block", "workload": workload + (", QK-RMSNorm" if args.qk_norm else ""),
                      "ms_per_block": ms, "block_tflops": tf,
                      "frac_of_bf16_burst": tf / peaks.get("bf16_tflops", 1900.0),
                      "skip_ms": ms_skip, "skip_gbs": gbs,
                      "skip_frac_of_hbm": gbs / peaks.get("hbm_gbs", 6800.0),
                      "peaks": src, "steps": args.steps, "warmup": args.warmup}))
    ctx.close()


def profile_mode(args):
    """One profiled sample (direct launches, only the taken branch launched) and its
    per-kernel-class split; the process an ncu launch list is taken on, because ncu
    does not profile kernels inside graphs that hold conditional nodes."""
    import torch

    from paper_2608_09231_gb300 import bag, configs, synth

    cfg = configs.get_config(args.config, guidance=args.guidance, qk_norm=args.qk_norm)
    T = args.T or cfg["T"]
    ctx = bag.create(cfg, T=T, B=args.budget)
    inp = synth.make_inputs(cfg)
    x = torch.from_numpy(inp["x"]).cuda()
    txt = torch.from_numpy(inp["txt"]).cuda()
    if cfg["dtype"] == "bf16":
        txt = txt.to(torch.bfloat16)
    pooled = torch.from_numpy(inp["pooled"]).cuda()
    unc = ()
    if args.guidance is not None:
        unc = (torch.from_numpy(inp["txt_u"]).cuda().to(txt.dtype),
               torch.from_numpy(inp["pooled_u"]).cuda())
    mask, _, nfe, prof = ctx.profile_run(x, txt, pooled, *unc)
    torch.cuda.synchronize()
    tot = sum(v["ms"] for v in prof.values())
    print(json.dumps({"mode": "profile", "config": args.config, "T": T, "B": args.budget,
                      "nfe": nfe, "mask": [int(m) for m in mask],
                      "kernels": {k: {"launches": v["launches"], "ms": round(v["ms"], 3),
                                      "share": round(v["ms"] / tot, 4)} for k, v in prof.items()}}))
    ctx.close()


def replica_barrier(world):
    """Barrier across the replicas (no-op for one process)."""
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(value, world, device=None):
    """The largest per-rank value (the job's time is its slowest replica's); works with
    any initialised process-group backend (NCCL for GPU tensors, gloo on the CPU)."""
    if world <= 1:
        return float(value)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_seconds_per_sample(ms_per_step_max, world):
    """Whole-job throughput as s/sample: every replica finishes one sample per step, so
    world samples take the slowest replica's step time."""
    return ms_per_step_max / 1e3 / world


def budget_overhead(sweep, prof, T):
    """How s/sample scales with the budget (the benchmark spec: with B/T plus a measured gate and
    skip overhead).  sweep: {B: s/sample}; prof: the profiled sample's per-class times.
    A least-squares line s(B) = slope * B + fixed over the swept budgets gives the cost of
    one more full step and the budget-independent part; the profiled sample gives the
    per-step cost of the method's own kernels (signal, gate, cache refresh / reuse)."""
    out = {}
    pts = sorted((int(b), float(v)) for b, v in sweep.items())
    if len(pts) >= 2:
        n = len(pts)
        mb = sum(b for b, _ in pts) / n
        mv = sum(v for _, v in pts) / n
        sxx = sum((b - mb) ** 2 for b, _ in pts)
        slope = sum((b - mb) * (v - mv) for b, v in pts) / sxx
        out["fit_ms_per_full_step"] = slope * 1e3
        out["fit_fixed_ms"] = (mv - slope * mb) * 1e3
        out["fit_max_residual_ms"] = max(abs(v - (mv + slope * (b - mb))) for b, v in pts) * 1e3
    total = sum(v["ms"] for v in prof.values())
    own = 0.0
    for k in ("signal", "gate", "cache"):
        if k in prof:
            out[f"{k}_us_per_step"] = prof[k]["ms"] * 1e3 / T
            own += prof[k]["ms"]
    if total > 0:
        out["method_kernels_share"] = own / total
    return out


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--budget", type=int, default=20)
    ap.add_argument("--config", default="flux")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-sweep", action="store_true")
    ap.add_argument("--mode", default="sample", choices=["sample", "block", "profile"])
    ap.add_argument("--T", type=int, default=0, help="profile mode: override the step count")
    ap.add_argument("--guidance", type=float, default=None,
                    help="classifier-free guidance scale (two branches, one shared mask)")
    ap.add_argument("--qk-norm", action="store_true",
                    help="per-head RMSNorm of q and k before RoPE (FLUX / Qwen-Image blocks)")
    args = ap.parse_args()
    if args.mode == "block":
        block_mode(args)
        return
    if args.mode == "profile":
        profile_mode(args)
        return
    ws, rank, local = _dist()

    from paper_2608_09231_gb300 import configs
    cfg = configs.get_config(args.config, guidance=args.guidance, qk_norm=args.qk_norm)
    B, T = args.budget, cfg["T"]
    workload = (f"{args.config}-shaped DiT, {cfg['n_double']} double + {cfg['n_single']} single "
                f"blocks, d={cfg['hidden']}, {cfg['n_img']} img + {cfg['n_txt']} txt tokens, "
                f"T={T}, B={B}, batch 1")
    if args.guidance is not None:
        workload += (f", classifier-free guidance g={args.guidance:g} (conditional and "
                     "unconditional branch, one shared mask)")
    if args.qk_norm:
        workload += ", QK-RMSNorm"
    config = {"workload": workload, "T": T, "B": B, "n_img": cfg["n_img"], "n_txt": cfg["n_txt"],
              "hidden": cfg["hidden"], "global_batch": ws, "seq_len": cfg["n_img"] + cfg["n_txt"],
              "parallelism": f"replicas x{ws}",
              "l2": "inputs larger than L2 (weights streamed every full step)"}

    if args.impl == "reference":
        if rank != 0:
            return
        res = run_cpu_oracle(args.config, args.steps, args.warmup)
        vals = [oracle_s_per_sample(cfg, B, r) for r in res["reps"]]
        v = statistics.mean(vals)
        line = {"impl": "reference", "metric": METRIC, "value": v, "unit": "s/sample",
                "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
                "ms_per_step": v * 1e3, "higher_is_better": False, "scaling": "weak",
                "vs_baseline": None, "dtype": "f64", "data": "synthetic", "config": config,
                "cpu_baseline": {"value": v, "unit": "s/sample", "cores": res["threads"],
                                 "kind": "oracle",
                                 "sample": "per step: one block of each kind in the stack, "
                                           "forward at full width and tokens in fp64, "
                                           "extrapolated linearly to B full stacks"},
                "e2e": {"value": v, "unit": "s/sample", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}}
        print(json.dumps(line))
        return

    import numpy as np
    import torch

    from paper_2608_09231_gb300 import bag, synth

    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    ctx = bag.create(cfg, T=T, B=B)
    stream = torch.cuda.current_stream()
    ctx.set_stream(stream.cuda_stream)
    inp = synth.make_inputs(cfg, sample_seed=rank)
    x0 = torch.from_numpy(inp["x"]).to(dev)
    txt = torch.from_numpy(inp["txt"]).to(dev)
    if cfg["dtype"] == "bf16":
        txt = txt.to(torch.bfloat16)
    pooled = torch.from_numpy(inp["pooled"]).to(dev)
    unc = ()
    if args.guidance is not None:
        unc = (torch.from_numpy(inp["txt_u"]).to(dev).to(txt.dtype),
               torch.from_numpy(inp["pooled_u"]).to(dev))
    x = torch.empty_like(x0)

    def one_sample():
        ctx.reset()
        x.copy_(x0)
        return ctx.run(x, txt, pooled, *unc)

    for _ in range(args.warmup):
        one_sample()
    torch.cuda.synchronize()

    def barrier():
        replica_barrier(ws)

    clocks = Clocks(local)
    clocks.start()
    barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    nfes, launches = [], 0
    for _ in range(args.steps):
        mask, log, nfe = one_sample()
        nfes.append(nfe)
        launches += ctx.launch_count()
    e1.record(stream)
    torch.cuda.synchronize()
    barrier()
    clk = clocks.stop()
    ms = e0.elapsed_time(e1) / args.steps
    ms = max_over_ranks(ms, ws, dev)
    s_per_sample = job_seconds_per_sample(ms, ws)
    assert all(n == B for n in nfes), nfes

    # end to end through the host-buffer entry point (pinned host memory)
    xh = torch.empty(x0.shape, dtype=torch.float32, pin_memory=True)
    txth = torch.from_numpy(inp["txt"].astype(np.float32)).pin_memory()
    pooledh = torch.from_numpy(inp["pooled"]).pin_memory()
    xh_np, txth_np, pooledh_np = xh.numpy(), txth.numpy(), pooledh.numpy()
    unch = ()
    if args.guidance is not None:
        unch = (torch.from_numpy(inp["txt_u"].astype(np.float32)).pin_memory(),
                torch.from_numpy(inp["pooled_u"]).pin_memory())
    unch_np = tuple(t.numpy() for t in unch)
    e2e_n = max(1, min(args.steps, 3))
    barrier()
    t0 = time.perf_counter()
    for _ in range(e2e_n):
        xh_np[...] = inp["x"]
        ctx.reset()
        ctx.run_host(xh_np, txth_np, pooledh_np, *unch_np)
    e2e_s = (time.perf_counter() - t0) / e2e_n
    e2e_s = max_over_ranks(e2e_s, ws, dev)
    h2d = x0.numel() * 4 + txth.numel() * 4 + pooledh.numel() * 4 + sum(t.numel() * 4 for t in unch)
    d2h = x0.numel() * 4 + T * (bag.LOG_FLOATS * 4 + 1) + 32

    # profiled sample: per-launch event timing (not part of the timed value)
    ctx.reset()
    x.copy_(x0)
    _, _, _, prof = ctx.profile_run(x, txt, pooled, *unc)
    recs = ctx.profile_launches()
    peaks, peak_src = _peaks()
    peak_t = peaks.get("bf16_tflops_sustained", 1700.0)
    roofline = dominant_roofline(recs, peaks, peak_src, args.config, f32=cfg["dtype"] == "f32")
    g, a = prof["gemm"], prof["attention"]
    gemm_tflops = g["flops"] / (g["ms"] * 1e-3) / 1e12 if g["ms"] > 0 else 0.0
    attn_tflops = a["flops"] / (a["ms"] * 1e-3) / 1e12 if a["ms"] > 0 else 0.0
    block_tflops = ((g["flops"] + a["flops"]) / ((g["ms"] + a["ms"]) * 1e-3) / 1e12
                    if g["ms"] + a["ms"] > 0 else 0.0)
    total_ms = sum(v["ms"] for v in prof.values())
    kernels = {}
    for k, v in prof.items():
        e = {"launches": v["launches"], "ms": round(v["ms"], 3),
             "share": round(v["ms"] / max(1e-9, total_ms), 4)}
        if v["ms"] > 0:
            if v["flops"]:
                e["tflops"] = round(v["flops"] / (v["ms"] * 1e-3) / 1e12, 1)
            else:
                e["gbs"] = round(v["bytes"] / (v["ms"] * 1e-3) / 1e9, 1)
        kernels[k] = e

    # budget sweep (context: how s/sample scales with B)
    sweep = {}
    if not args.no_sweep and rank == 0:
        for Bs in cfg["budgets"]:
            if Bs == B:
                sweep[str(Bs)] = s_per_sample
                continue
            c2 = bag.create(cfg, T=T, B=Bs)
            c2.set_stream(stream.cuda_stream)
            c2.reset()
            x.copy_(x0)
            c2.run(x, txt, pooled, *unc)
            torch.cuda.synchronize()
            f0, f1 = torch.cuda.Event(True), torch.cuda.Event(True)
            f0.record(stream)
            c2.reset()
            x.copy_(x0)
            c2.run(x, txt, pooled, *unc)
            f1.record(stream)
            torch.cuda.synchronize()
            sweep[str(Bs)] = f0.elapsed_time(f1) / 1e3
            c2.close()

    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        try:
            res = run_cpu_oracle(args.config, 1, 0)
            rep = res["reps"][0]
            cpu = {"value": oracle_s_per_sample(cfg, B, rep), "unit": "s/sample",
                   "cores": res["threads"], "kind": "oracle",
                   "sample": ("one block of each kind at full width/tokens in fp64 ("
                              + ", ".join(f"{k[:-2]} {v:.2f} s" for k, v in rep.items() if v)
                              + f"), extrapolated to B={B} full stacks")}
        except Exception as ex:  # reported, never silently replaced
            cpu = {"value": None, "unit": "s/sample", "cores": os.cpu_count(), "kind": "oracle",
                   "sample": f"failed: {ex}"}

    if rank == 0:
        line = {"metric": METRIC, "value": s_per_sample, "unit": "s/sample", "n_gpus": ws,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
                "higher_is_better": False, "scaling": "weak",
                "vs_baseline": (s_per_sample / PAPER_S_PER_SAMPLE[B]
                                if B in PAPER_S_PER_SAMPLE and args.config == "flux"
                                and args.guidance is None else None),
                "dtype": cfg["dtype"], "data": "synthetic (seeded random weights and inputs)",
                "config": config, "clocks": clk,
                "e2e": {"value": e2e_s / ws, "unit": "s/sample", "h2d_bytes_per_step": h2d,
                        "d2h_bytes_per_step": d2h},
                "gpu_launches": launches, "roofline": roofline,
                "dit_block_tflops": {"value": block_tflops, "gemm": gemm_tflops,
                                     "attention": attn_tflops, "peak": peak_t,
                                     "frac": block_tflops / peak_t},
                "kernels": kernels, "budget_sweep_s_per_sample": sweep,
                "overhead": budget_overhead(sweep, prof, T),
                "cpu_baseline": cpu}
        print(json.dumps(line))
    ctx.close()
    if ws > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    if len(sys.argv) > 1 and sys.argv[1] == "--cpu-worker":
        cpu_worker(sys.argv[2], int(sys.argv[3]), int(sys.argv[4]))
    else:
        main()
