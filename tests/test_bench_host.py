"""Host-side arithmetic of the benchmark (no GPU): the algorithmic work it divides by,
the roofline of the dominant kernel group, and whole-job throughput over replicas."""

import importlib.util
import os
import sys

import pytest

from paper_2608_09231_gb300 import configs

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    argv = sys.argv
    sys.argv = ["bench.py"]
    try:
        spec.loader.exec_module(mod)
    finally:
        sys.argv = argv
    return mod


@pytest.mark.parametrize("name,tflop", [("flux", 74.36), ("qwen", 134.74), ("wan", 1678.3)])
def test_block_flops_add_up_to_a_forward(bench, name, tflop):
    """Per-forward work of the three stacks (2·M·N·K per projection, 4·n_q·n_k·d per
    attention): FLUX 74.36, Qwen-Image 134.74, Wan2.1-14B ≈ 1678 TFLOP."""
    cfg = configs.get_config(name)
    total = 0.0
    for kind, n in (("double", cfg["n_double"]), ("single", cfg["n_single"]), ("wan", cfg["n_wan"])):
        if n == 0:
            continue
        over = {"n_double": 0, "n_single": 0, "n_wan": 0}
        over["n_" + kind] = 1
        total += n * bench.block_flops(configs.get_config(name, **over))
    assert abs(total / 1e12 - tflop) <= 1e-3 * tflop, total / 1e12


def test_flux_blocks_have_equal_work(bench):
    """A FLUX double-stream block and a single-stream block do the same flops (both
    project the joint sequence to 3d + F and back)."""
    d = configs.get_config("flux", n_double=1, n_single=0)
    s = configs.get_config("flux", n_double=0, n_single=1)
    assert abs(bench.block_flops(d) - bench.block_flops(s)) <= 1e-9 * bench.block_flops(s)


def test_dominant_roofline_picks_the_costliest_group(bench):
    recs = ([{"kind": "gemm", "m": 4608, "n": 21504, "k": 3072, "variant": 1, "ms": 0.36,
              "flops": 2.0 * 4608 * 21504 * 3072, "bytes": 0.0}] * 3 +
            [{"kind": "attention", "m": 4608, "n": 4608, "k": 24, "variant": 0, "ms": 0.2,
              "flops": 4.0 * 4608 * 4608 * 24 * 128, "bytes": 0.0}] * 4 +
            [{"kind": "norm", "m": 4608, "n": 3072, "k": 0, "variant": 0, "ms": 0.02,
              "flops": 0.0, "bytes": 4608 * 3072 * 6.0}] * 20)
    r = bench.dominant_roofline(recs, {"bf16_tflops_sustained": 1700.0}, "measured", "flux")
    assert r["kernel"] == "gemm_pair_kernel" and r["shape"] == [4608, 21504, 3072]
    assert r["bound"] == "tensor" and r["launches"] == 3
    want = 2.0 * 4608 * 21504 * 3072 / 0.36e-3 / 1e12
    assert abs(r["achieved"] - want) <= 1e-9 * want and abs(r["frac"] - want / 1700.0) < 1e-12
    assert abs(r["share_of_profiled_time"] - 1.08 / (1.08 + 0.8 + 0.4)) < 1e-12
    # a memory-bound group is measured in GB/s against the copy bandwidth
    r = bench.dominant_roofline(recs[-20:], {"hbm_gbs": 6760.0}, "measured", "flux")
    assert r["bound"] == "hbm" and r["unit"] == "GB/s"
    assert abs(r["achieved"] - 4608 * 3072 * 6.0 / 0.02e-3 / 1e9) < 1e-6


def test_job_throughput_counts_every_replica(bench):
    # N replicas finish N samples in the slowest replica's step time
    assert bench.job_seconds_per_sample(1000.0, 1) == 1.0
    assert bench.job_seconds_per_sample(1000.0, 4) == 0.25


def test_budget_overhead_fit(bench):
    """The budget fit recovers an exact line s(B) = 0.05 B + 0.02 and the per-step cost of
    the method's own kernels from the profiled classes."""
    sweep = {str(b): 0.05 * b + 0.02 for b in (25, 20, 15, 10)}
    prof = {"gemm": {"ms": 900.0}, "attention": {"ms": 80.0}, "signal": {"ms": 2.0},
            "gate": {"ms": 1.0}, "cache": {"ms": 1.5}, "norm": {"ms": 15.5}}
    o = bench.budget_overhead(sweep, prof, 50)
    assert abs(o["fit_ms_per_full_step"] - 50.0) < 1e-9
    assert abs(o["fit_fixed_ms"] - 20.0) < 1e-9 and o["fit_max_residual_ms"] < 1e-9
    assert abs(o["signal_us_per_step"] - 40.0) < 1e-9 and abs(o["gate_us_per_step"] - 20.0) < 1e-9
    assert abs(o["method_kernels_share"] - 4.5 / 1000.0) < 1e-12
    assert "fit_ms_per_full_step" not in bench.budget_overhead({"20": 1.0}, prof, 50)
