"""The allocation-free signal entry point (bag_rel_l1_noalloc).

Some callers cannot call cudaMalloc (a host framework's caching allocator owns the
device memory, or the loop cannot take cudaMalloc's implicit synchronisation), so they
cannot create a context either.  bag_rel_l1_noalloc serves them with its scratch in a
fixed device array of the library.  This test checks it through the C ABI against the
regular entry point (bag_rel_l1, caller-provided scratch) on two calls in a row, which
share that array, and checks the size limit.  The file sorts last so that a run which
stops at the first failure has already run every other test.
"""

import numpy as np
import pytest
import torch

from paper_2608_09231_gb300 import bag, synth

pytestmark = pytest.mark.gpu


def _pair(seed, rows, cols, bf16):
    a = synth.normal(seed, 1, rows * cols, 1.0).reshape(rows, cols)
    b = a + synth.normal(seed, 2, rows * cols, 0.1 * seed).reshape(rows, cols)
    dt = torch.bfloat16 if bf16 else torch.float32
    return torch.from_numpy(a).cuda().to(dt), torch.from_numpy(b).cuda().to(dt)


def test_noalloc_matches_scratch_entry_point_twice(lib):
    ctx = bag.create("tiny", T=2, B=1)
    stream = torch.cuda.current_stream().cuda_stream
    # two calls in a row with different sizes: the second must not see the first's rows
    for seed, rows, cols, bf16 in [(3, 4096, 3072, 1), (5, 300, 256, 0)]:
        A, B = _pair(seed, rows, cols, bf16)
        scratch = torch.empty(2 * rows, dtype=torch.float32, device="cuda")
        want = torch.empty(3, dtype=torch.float32, device="cuda")
        got = torch.full((3,), float("nan"), dtype=torch.float32, device="cuda")
        ctx.rel_l1(A, B, rows, cols, scratch, want)
        torch.cuda.synchronize()
        bag.rel_l1_noalloc(A, B, rows, cols, got, stream)
        torch.cuda.synchronize()
        w, g = want.cpu().numpy(), got.cpu().numpy()
        assert np.all(np.isfinite(g))
        assert np.allclose(g, w, rtol=1e-5, atol=0.0), (g, w)
    ctx.close()


def test_noalloc_rejects_rows_beyond_limit(lib):
    x = torch.zeros((65537, 4), dtype=torch.float32, device="cuda")
    out = torch.empty(3, dtype=torch.float32, device="cuda")
    with pytest.raises(bag.BagError) as ei:
        bag.rel_l1_noalloc(x, x, 65537, 4, out, torch.cuda.current_stream().cuda_stream)
    assert ei.value.status == 1 and "65536" in str(ei.value)
