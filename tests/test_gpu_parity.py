"""GPU path against the fp64 oracle, through the C ABI.

Bars (from the method's arithmetic):
  * schedules: the full/cached bit of every step is bit-exact when the oracle takes its
    decisions on the GPU's logged gate inputs; the gate logit itself is bit-exact
    (both sides evaluate it in fp32 in the same order);
  * latents: max-abs error <= 1e-4 x RMS(oracle) for the fp32 configuration and
    <= 2e-2 x RMS(oracle) for bf16 configurations;
  * integer/byte work (weights from the seeded generator, NFE counts) bit-exact.
"""

import numpy as np
import pytest
import torch

from oracle import bag_oracle as O
from paper_2608_09231_gb300 import bag, configs, synth

pytestmark = pytest.mark.gpu

TOL = {"f32": 1e-4, "bf16": 2e-2}


def _dev_inputs(cfg, inp):
    x = torch.from_numpy(inp["x"].copy()).cuda()
    txt = torch.from_numpy(inp["txt"]).cuda()
    if cfg["dtype"] == "bf16":
        txt = txt.to(torch.bfloat16)
    pooled = torch.from_numpy(inp["pooled"]).cuda()
    return x, txt, pooled


def _gpu_sample(cfg, T, B, tau=0.5, policy=None, mask=None, ctx=None, delta=0.0):
    own = ctx is None
    if own:
        ctx = bag.create(cfg, T=T, B=B, tau=tau)
    inp = synth.make_inputs(cfg)
    x, txt, pooled = _dev_inputs(cfg, inp)
    if policy is not None:
        ctx.set_policy(policy, mask, delta)
    ctx.reset()
    m, log, nfe = ctx.run(x, txt, pooled)
    torch.cuda.synchronize()
    out = x.cpu().numpy()
    if own:
        ctx.close()
    return inp, out, m, log, nfe


def _gate_inputs(log):
    return [None] + [float(v) for v in log[1:, 2]]


@pytest.mark.parametrize("name", ["tiny", "flux_small", "wan_small"])
def test_device_weights_equal_generator(name, lib):
    cfg = configs.get_config(name)
    ctx = bag.create(cfg, T=4, B=2)
    W = synth.make_weights(cfg)
    for blk, tname in [(-1, "pe_w"), (-1, "fin_b"), (-1, "t1_w"), (0, W["blocks"][0] and
                                                                  list(W["blocks"][0])[1]),
                       (len(W["blocks"]) - 1, list(W["blocks"][-1])[-1])]:
        ref = W["global"][tname] if blk < 0 else W["blocks"][blk][tname]
        got = ctx.get_weight(blk, tname, ref.size).reshape(ref.shape)
        assert np.array_equal(got, ref), (blk, tname)
    ctx.close()


@pytest.mark.parametrize("name", ["tiny", "tiny_ragged", "single_small", "flux_small",
                                  "qwen_small", "wan_small"])
def test_sample_parity_against_oracle(name, lib):
    cfg = configs.get_config(name)
    T, B = cfg["T"], cfg["budgets"][0]
    inp, got, mask, log, nfe = _gpu_sample(cfg, T, B)
    assert nfe == B and int(mask.sum()) == B and mask[0] == 1
    W = synth.make_weights(cfg)
    g = synth.make_gate(cfg["gate_seed"])
    ref = O.sample(cfg, W, g, inp, T=T, B=B, drift_override=_gate_inputs(log))
    # schedule bit-exact, gate logit bit-exact on the GPU's inputs
    assert list(mask) == ref["mask"]
    for t in range(1, T):
        f = [np.float32(v) for v in log[t, 0:3]]
        assert O.gate_logit(f, g) == np.float32(log[t, 3]), t
        assert f[0] == np.float32(B - log[t, 6]) / np.float32(B)
        assert f[1] == np.float32(T - t) / np.float32(T)
        # the GPU's drift agrees with the oracle's own drift
        dref = ref["log"][t]["drift"]
        assert abs(float(log[t, 2]) - dref) <= max(TOL[cfg["dtype"]], 1e-6) * max(dref, 1e-3), t
    rms = float(np.sqrt(np.mean(ref["x"] ** 2)))
    err = float(np.max(np.abs(got.astype(np.float64) - ref["x"])))
    assert err <= TOL[cfg["dtype"]] * rms, (err, rms)


@pytest.mark.parametrize("name", ["tiny", "flux_small"])
def test_budget_equal_T_is_uncached_sampling_bit_exact(name, lib):
    cfg = configs.get_config(name)
    T = 5
    _, a, ma, _, na = _gpu_sample(cfg, T, T)
    _, b, mb, _, nb = _gpu_sample(cfg, T, 1, policy=bag.POLICY_FULL)
    assert na == nb == T and list(ma) == list(mb) == [1] * T
    assert np.array_equal(a, b)


@pytest.mark.parametrize("tau", [0.3, 0.5, 0.7])
def test_nfe_equals_budget_for_any_tau(tau, lib):
    cfg = configs.get_config("tiny_ragged")
    T = cfg["T"]
    for B in (1, 3, T):
        _, _, m, log, nfe = _gpu_sample(cfg, T, B, tau=tau)
        assert nfe == B and int(m.sum()) == B and m[0] == 1
        assert list(m) == O.schedule_from_gate_bits([None] + [int(v) for v in log[1:, 4]], B, T)


def test_static_mask_policy(lib):
    cfg = configs.get_config("tiny_ragged")
    T = cfg["T"]
    want = [1, 0, 1, 1, 0, 0, 1]
    _, got, m, _, nfe = _gpu_sample(cfg, T, 4, policy=bag.POLICY_MASK, mask=np.array(want, np.uint8))
    assert list(m) == want and nfe == 4
    inp = synth.make_inputs(cfg)
    ref = O.sample(cfg, synth.make_weights(cfg), synth.make_gate(cfg["gate_seed"]), inp, T=T, B=4,
                   policy=want)
    rms = float(np.sqrt(np.mean(ref["x"] ** 2)))
    assert float(np.max(np.abs(got - ref["x"]))) <= TOL["f32"] * rms


@pytest.mark.parametrize("name", ["tiny", "flux_small"])
def test_step_api_matches_run(name, lib):
    cfg = configs.get_config(name)
    T, B = 6, 3
    ctx = bag.create(cfg, T=T, B=B)
    inp = synth.make_inputs(cfg)
    x, txt, pooled = _dev_inputs(cfg, inp)
    x0 = x.clone()
    m_run, _, _ = ctx.run(x, txt, pooled)
    ctx.reset()
    xs = x0.clone()
    flags = torch.zeros(T, dtype=torch.int32, device="cuda")
    with pytest.raises(bag.BagError) as ei:
        ctx.step(xs, 1, txt, pooled, xs, flags[1:])
    assert ei.value.status == 4  # EORDER
    for t in range(T):
        ctx.step(xs, t, txt, pooled, xs, flags[t:])
    torch.cuda.synchronize()
    assert list(flags.cpu().numpy()) == list(m_run)
    assert torch.equal(xs, x)
    ctx.close()


def test_run_host_matches_device(lib):
    cfg = configs.get_config("flux_small")
    T, B = 5, 3
    ctx = bag.create(cfg, T=T, B=B)
    inp = synth.make_inputs(cfg)
    x, txt, pooled = _dev_inputs(cfg, inp)
    m1, _, _ = ctx.run(x, txt, pooled)
    ctx.reset()
    xh = inp["x"].copy()
    m2, _, _ = ctx.run_host(xh, inp["txt"], inp["pooled"])
    assert list(m1) == list(m2)
    assert np.array_equal(xh, x.cpu().numpy())
    ctx.close()


# ---------------------------------------------------------------------------
# kernel-level parity
# ---------------------------------------------------------------------------
def _bf16_tensor(seed, shape, std=1.0):
    v = synth.bf16_round(synth.normal(seed, 77, int(np.prod(shape)), std)).reshape(shape)
    return v, torch.from_numpy(v).cuda().to(torch.bfloat16)


# (4096, 3072, 3072), (1000, 19456, 192), (4100, 4864, 320) and (7000, 3072, 256) have
# enough 256 x 256 tiles for the CTA-pair kernel (the last three with a ragged final row
# tile); (50, 38912, 256) is less than one tile high and wide enough for the pair kernel
# (the shape class of the per-sample modulation GEMM, M = T)
@pytest.mark.parametrize("M,N,K", [(300, 256, 128), (129, 64, 64), (1000, 384, 512),
                                   (77, 512, 256), (4096, 3072, 3072), (50, 1024, 320),
                                   (1000, 19456, 192), (4100, 4864, 320), (7000, 3072, 256),
                                   (50, 38912, 256)])
@pytest.mark.parametrize("simt", [0, 1])
def test_gemm_bf16_against_fp64(M, N, K, simt, lib):
    ctx = bag.create("tiny", T=2, B=1)
    a, A = _bf16_tensor(1, (M, K))
    w, Wt = _bf16_tensor(2, (N, K), 0.05)
    b = synth.normal(3, 5, N, 0.1)
    bias = torch.from_numpy(b).cuda()
    C = torch.zeros((M, N), dtype=torch.float32, device="cuda")
    ctx.gemm_bf16(A, Wt, bias, C, M, N, K, 0, simt)
    torch.cuda.synchronize()
    rows = np.arange(M) if M * N <= 1100 * 4096 else np.r_[0:64, M - 64:M, 500:510]
    ref = a[rows].astype(np.float64) @ w.T.astype(np.float64) + b
    bound = 4 * K * 2.0 ** -24 * (np.abs(a[rows]).astype(np.float64) @ np.abs(w).T) + 1e-7
    got = C.cpu().numpy()[rows]
    assert np.all(np.abs(got - ref) <= bound)
    ctx.close()


@pytest.mark.parametrize("M,N,K", [(257, 128, 192), (700, 19456, 128), (7000, 3072, 128)])
def test_gemm_gelu_epilogue(M, N, K, lib):
    ctx = bag.create("tiny", T=2, B=1)
    a, A = _bf16_tensor(4, (M, K))
    w, Wt = _bf16_tensor(5, (N, K), 0.1)
    C = torch.zeros((M, N), dtype=torch.float32, device="cuda")
    ctx.gemm_bf16(A, Wt, None, C, M, N, K, 1, 0)
    torch.cuda.synchronize()
    ref = O.gelu_tanh(a.astype(np.float64) @ w.T.astype(np.float64))
    assert np.max(np.abs(C.cpu().numpy() - ref)) <= 1e-4 * (1 + np.max(np.abs(ref)))
    ctx.close()


@pytest.mark.parametrize("rows,cols", [(37, 256), (1000, 3072), (5, 5120), (3655, 3072), (20000, 256)])
def test_ln_mod_against_oracle(rows, cols, lib):
    ctx = bag.create("tiny", T=2, B=1)
    x = synth.normal(7, 1, rows * cols, 2.0).reshape(rows, cols) + 0.5
    sh = synth.normal(7, 2, cols, 0.5)
    sc = synth.normal(7, 3, cols, 0.5)
    y = torch.zeros((rows, cols), dtype=torch.bfloat16, device="cuda")
    ctx.ln_mod(torch.from_numpy(x).cuda(), torch.from_numpy(sh).cuda(),
               torch.from_numpy(sc).cuda(), y, rows, cols)
    torch.cuda.synchronize()
    ref = O.modulate(O.layer_norm(x.astype(np.float64)), sh, sc)
    got = y.float().cpu().numpy()
    assert np.all(np.abs(got - ref) <= 2.0 ** -8 * np.abs(ref) + 1e-5)
    ctx.close()


@pytest.mark.parametrize("rows,cols,bf16", [(4096, 3072, 1), (37, 256, 0), (1, 64, 1)])
def test_rel_l1_against_oracle(rows, cols, bf16, lib):
    ctx = bag.create("tiny", T=2, B=1)
    a = synth.normal(21, 1, rows * cols, 1.0).reshape(rows, cols)
    b = a + synth.normal(21, 2, rows * cols, 0.05).reshape(rows, cols)
    if bf16:
        a, b = synth.bf16_round(a), synth.bf16_round(b)
    dt = torch.bfloat16 if bf16 else torch.float32
    A = torch.from_numpy(a).cuda().to(dt)
    Bt = torch.from_numpy(b).cuda().to(dt)
    scratch = torch.empty(2 * rows, dtype=torch.float32, device="cuda")
    out = torch.empty(3, dtype=torch.float32, device="cuda")
    ctx.rel_l1(A, Bt, rows, cols, scratch, out)
    torch.cuda.synchronize()
    ref = O.rel_l1(a.astype(np.float64), b.astype(np.float64))
    got = out.cpu().numpy()
    assert abs(float(got[0]) - ref) <= 1e-5 * ref
    assert abs(float(got[2]) - np.abs(b.astype(np.float64)).sum()) <= 1e-5 * float(got[2])
    # identical inputs give exactly zero
    ctx.rel_l1(Bt, Bt, rows, cols, scratch, out)
    torch.cuda.synchronize()
    assert float(out[0].item()) == 0.0
    ctx.close()


def test_empty_inputs_are_no_ops_and_undefined_ones_are_rejected(lib):
    """Zero rows (GEMM, LN-mod), zero queries (attention) and zero elements (residual
    add) launch nothing and leave every output untouched; a relative L1 over no rows and
    an attention over no keys have no value and are refused with EINVAL."""
    ctx = bag.create("tiny", T=2, B=1)
    bf = torch.bfloat16
    C = torch.full((4, 64), 7.0, device="cuda")
    ctx.gemm_bf16(torch.zeros((1, 64), dtype=bf, device="cuda"),
                  torch.zeros((64, 64), dtype=bf, device="cuda"), None, C, 0, 64, 64)
    x = torch.zeros((1, 256), device="cuda")
    y = torch.full((1, 256), 7.0, dtype=bf, device="cuda")
    ctx.ln_mod(x, torch.zeros(256, device="cuda"), torch.zeros(256, device="cuda"), y, 0, 256)
    q = torch.zeros((1, 256), dtype=bf, device="cuda")
    kv = torch.zeros((16, 256), dtype=bf, device="cuda")
    o = torch.full((1, 256), 7.0, dtype=bf, device="cuda")
    ctx.attention_bf16(q, kv, kv, o, 0, 16, 4, 64, 0, 1)
    r = torch.full((8,), 7.0, device="cuda")
    ctx.residual_add(r, torch.zeros(8, device="cuda"), torch.zeros(8, device="cuda"), 0)
    torch.cuda.synchronize()
    for t in (C, y, o, r):
        assert bool(torch.all(t.float() == 7.0))
    scratch = torch.empty(2, device="cuda")
    out = torch.full((3,), 7.0, device="cuda")
    with pytest.raises(bag.BagError) as ei:
        ctx.rel_l1(x, x, 0, 256, scratch, out)
    assert bag.STATUS[ei.value.status] == "BAG_EINVAL"
    with pytest.raises(bag.BagError):
        ctx.attention_bf16(q, kv, kv, o, 1, 0, 4, 64, 0, 1)
    torch.cuda.synchronize()
    assert bool(torch.all(out == 7.0)) and bool(torch.all(o.float() == 7.0))
    ctx.close()


@pytest.mark.parametrize("name", ["tiny", "flux_small"])
def test_single_step_sample(name, lib):
    """T = 1 (so B = 1): the one step is computed in full (Algorithm 2's forced first
    step) and the sample is one uncached Euler step from sigma = 1 to 0."""
    cfg = configs.get_config(name)
    inp, out, m, log, nfe = _gpu_sample(cfg, 1, 1)
    assert nfe == 1 and list(m) == [1]
    W, g = synth.make_weights(cfg), synth.make_gate(cfg["gate_seed"])
    ref = O.sample(cfg, W, g, inp, T=1, B=1)
    rms = float(np.sqrt(np.mean(ref["x"] ** 2)))
    assert list(ref["mask"]) == [1]
    assert float(np.max(np.abs(out - ref["x"]))) <= TOL[cfg["dtype"]] * rms


def test_calls_out_of_state_are_refused_and_leave_the_context_usable(lib):
    """ESTATE: a whole-sample call on a context whose sample is under way (or finished)
    until bag_reset, and a block forward before bag_prepare; EORDER: a step past T.
    After each refusal the context still samples, and equals a fresh context's sample."""
    cfg = configs.get_config("tiny")
    T, B = 3, 2
    ctx = bag.create(cfg, T=T, B=B)
    inp = synth.make_inputs(cfg)
    x, txt, pooled = _dev_inputs(cfg, inp)
    h = torch.zeros((cfg["n_txt"] + 256, cfg["hidden"]), device="cuda")
    with pytest.raises(bag.BagError) as ei:
        ctx.forward_block(0, 0, h)
    assert bag.STATUS[ei.value.status] == "BAG_ESTATE"
    x1 = x.clone()
    ctx.step(x1, 0, txt, pooled, x1)
    with pytest.raises(bag.BagError) as ei:
        ctx.run(x1, txt, pooled)
    assert bag.STATUS[ei.value.status] == "BAG_ESTATE"
    for t in range(1, T):
        ctx.step(x1, t, txt, pooled, x1)
    with pytest.raises(bag.BagError) as ei:
        ctx.step(x1, T, txt, pooled, x1)
    assert bag.STATUS[ei.value.status] == "BAG_EORDER"
    with pytest.raises(bag.BagError) as ei:
        ctx.run(x1, txt, pooled)
    assert bag.STATUS[ei.value.status] == "BAG_ESTATE"
    ctx.reset()
    x2 = x.clone()
    m2, _, n2 = ctx.run(x2, txt, pooled)
    torch.cuda.synchronize()
    _, ref, mr, _, nr = _gpu_sample(cfg, T, B)
    assert n2 == nr == B and list(m2) == list(mr)
    assert np.array_equal(x2.cpu().numpy(), ref) and torch.equal(x1, x2)
    ctx.close()


def test_residual_add_exact(lib):
    ctx = bag.create("tiny", T=2, B=1)
    n = 1 << 20
    a = torch.from_numpy(synth.normal(9, 1, n, 1.0)).cuda()
    r = torch.from_numpy(synth.normal(9, 2, n, 0.3)).cuda()
    out = torch.empty_like(a)
    ctx.residual_add(out, a, r, n)
    torch.cuda.synchronize()
    assert np.array_equal(out.cpu().numpy(), a.cpu().numpy() + r.cpu().numpy())
    ctx.close()


# the tensor-core kernel takes 256 query rows per CTA (ragged 1100 and 129 leave most of
# the last CTA's rows empty; 77 keys are one masked key tile)
@pytest.mark.parametrize("nq,nk,heads,dh", [(300, 300, 2, 128), (129, 515, 3, 128),
                                            (288, 288, 4, 64), (4608, 4608, 1, 128),
                                            (1100, 700, 2, 128), (2048, 77, 3, 128)])
@pytest.mark.parametrize("simt", [0, 1])
def test_attention_against_oracle(nq, nk, heads, dh, simt, lib):
    ctx = bag.create("tiny", T=2, B=1)
    d = heads * dh
    q, Q = _bf16_tensor(11, (nq, d))
    k, K_ = _bf16_tensor(12, (nk, d))
    v, V = _bf16_tensor(13, (nk, d))
    o = torch.zeros((nq, d), dtype=torch.bfloat16, device="cuda")
    if dh == 128:
        vpad = (nk + 127) // 128 * 128
        vt = torch.zeros((heads, dh, vpad), dtype=torch.bfloat16, device="cuda")
        vt[:, :, :nk] = V.reshape(nk, heads, dh).permute(1, 2, 0)
        ctx.attention_bf16(Q, K_, vt, o, nq, nk, heads, dh, vpad, simt)
    else:
        ctx.attention_bf16(Q, K_, V, o, nq, nk, heads, dh, 0, 1)
    torch.cuda.synchronize()
    rows = np.arange(nq) if nq <= 600 else np.r_[0:40, 250:290, 500:540, nq - 40:nq]
    ref = O.attention(q.reshape(nq, heads, dh).astype(np.float64),
                      k.reshape(nk, heads, dh).astype(np.float64),
                      v.reshape(nk, heads, dh).astype(np.float64), q_rows=rows).reshape(len(rows), d)
    got = o.float().cpu().numpy()[rows]
    # P and O are rounded to bf16: allow 2^-7 relative to the output scale
    assert np.max(np.abs(got - ref)) <= 2.0 ** -7 * (np.max(np.abs(ref)) + 1e-3)
    ctx.close()


@pytest.mark.parametrize("nq,nk,heads", [(300, 300, 2), (129, 515, 3), (4608, 4608, 1),
                                         (1100, 700, 2), (2048, 77, 3)])
def test_attention_f16_operands_against_oracle(nq, nk, heads, lib):
    """The operand type the sampling path uses: fp16 q, k, v (and P), bf16 output.  With
    11-bit operands the error is the output's bf16 rounding (<= 2^-8 relative) plus a small
    share from the fp16 P and operand roundings."""
    ctx = bag.create("tiny", T=2, B=1)
    dh = 128
    d = heads * dh

    def f16(seed, shape):
        v = synth.normal(seed, 77, int(np.prod(shape)), 1.0).reshape(shape).astype(np.float16)
        return v.astype(np.float64), torch.from_numpy(v).cuda()

    q, Q = f16(21, (nq, d))
    k, K_ = f16(22, (nk, d))
    v, V = f16(23, (nk, d))
    o = torch.zeros((nq, d), dtype=torch.bfloat16, device="cuda")
    vpad = (nk + 127) // 128 * 128
    vt = torch.zeros((heads, dh, vpad), dtype=torch.float16, device="cuda")
    vt[:, :, :nk] = V.reshape(nk, heads, dh).permute(1, 2, 0)
    ctx.attention_f16(Q, K_, vt, o, nq, nk, heads, dh, vpad)
    torch.cuda.synchronize()
    rows = np.arange(nq) if nq <= 600 else np.r_[0:40, 250:290, 500:540, nq - 40:nq]
    ref = O.attention(q.reshape(nq, heads, dh), k.reshape(nk, heads, dh),
                      v.reshape(nk, heads, dh), q_rows=rows).reshape(len(rows), d)
    got = o.float().cpu().numpy()[rows]
    assert np.max(np.abs(got - ref)) <= 1.2 * 2.0 ** -8 * (np.max(np.abs(ref)) + 1e-3)
    # elementwise: each output within its own bf16 rounding plus the fp16 share
    assert np.all(np.abs(got - ref) <= 2.0 ** -8 * np.abs(ref) + 2.0 ** -10 * np.max(np.abs(ref)))
    ctx.close()


# ---------------------------------------------------------------------------
# the paper's six-input gates (App. A.2) on all six scalars of Eq. 3
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("name,kind", [("flux_small", "flux6"), ("qwen_small", "wan6"),
                                       ("wan_small", "flux6"), ("tiny_ragged", "wan6")])
def test_six_input_gate_sample_parity(name, kind, lib):
    cfg = configs.get_config(name, gate_kind=kind)
    T, B = cfg["T"], cfg["budgets"][0]
    inp, got, mask, log, nfe = _gpu_sample(cfg, T, B)
    assert nfe == B and int(mask.sum()) == B and mask[0] == 1
    g = synth.make_gate6(cfg["gate_seed"], kind)
    ref = O.sample(cfg, synth.make_weights(cfg), g, inp, T=T, B=B,
                   drift_override=_gate_inputs(log),
                   step_override=[None] + [float(v) for v in log[1:, 13]])
    assert list(mask) == ref["mask"]
    tol = TOL[cfg["dtype"]]
    for t in range(1, T):
        c = int(log[t, 6])
        t_last = t - int(log[t, 7])
        f = O.gate_features6(B, T, c, t, t_last, float(log[t, 2]), float(log[t, 13]))
        assert [np.float32(v) for v in log[t, 8:11]] == f[:3], t
        assert O.gate_logit6(f, g) == np.float32(log[t, 3]), t
        sref = ref["log"][t]["s_traj"][2]
        assert abs(float(log[t, 13]) - sref) <= max(tol, 1e-6) * max(sref, 1e-3), t
    rms = float(np.sqrt(np.mean(ref["x"] ** 2)))
    assert float(np.max(np.abs(got.astype(np.float64) - ref["x"]))) <= tol * rms


@pytest.mark.parametrize("name,kind", [("flux_small", "flux6"), ("wan_small", "wan6"),
                                       ("tiny_ragged", "mlp3"), ("qwen_small", "flux6")])
def test_embedded_observable_sample_parity(name, kind, lib):
    """The paper's observable (Eq. 3): the signal reads the post-patch-embedding tokens.
    Schedules bit-exact on the GPU's logged gate inputs, the GPU's drift and step change
    equal the oracle's own within the dtype's bar, and the latent within its bar."""
    cfg = configs.get_config(name, gate_kind=kind, observable="embedded")
    T, B = cfg["T"], cfg["budgets"][0]
    inp, got, mask, log, nfe = _gpu_sample(cfg, T, B)
    assert nfe == B and int(mask.sum()) == B and mask[0] == 1
    g = synth.make_gate_any(cfg["gate_seed"], kind)
    ref = O.sample(cfg, synth.make_weights(cfg), g, inp, T=T, B=B,
                   drift_override=_gate_inputs(log),
                   step_override=[None] + [float(v) for v in log[1:, 13]])
    assert list(mask) == ref["mask"]
    # fp32 observable from a split-precision patch embedding: the drift carries only fp32
    # rounding (the latent itself differs by the dtype's bar, so allow that share)
    tol = max(TOL[cfg["dtype"]], 1e-6)
    for t in range(1, T):
        dref, sref = ref["log"][t]["drift"], ref["log"][t]["s_traj"][2]
        assert abs(float(log[t, 2]) - dref) <= tol * max(dref, 1e-3), t
        assert abs(float(log[t, 13]) - sref) <= tol * max(sref, 1e-3), t
        if kind == "mlp3":
            assert O.gate_logit([np.float32(v) for v in log[t, 0:3]], g) == np.float32(log[t, 3])
        else:
            f = O.gate_features6(B, T, int(log[t, 6]), t, t - int(log[t, 7]), float(log[t, 2]),
                                 float(log[t, 13]))
            assert O.gate_logit6(f, g) == np.float32(log[t, 3]), t
    rms = float(np.sqrt(np.mean(ref["x"] ** 2)))
    assert float(np.max(np.abs(got.astype(np.float64) - ref["x"]))) <= TOL[cfg["dtype"]] * rms
    # the GPU read the embedded observable: on the same schedule its drifts are closer to
    # the oracle's embedded drifts than to the drifts of the default (modulated) observable
    mod = O.sample(configs.get_config(name, gate_kind=kind), synth.make_weights(cfg), g, inp,
                   T=T, B=B, policy=ref["mask"])
    gpu = np.array([float(v) for v in log[1:, 2]])
    emb = np.array([ref["log"][t]["drift"] for t in range(1, T)])
    other = np.array([mod["log"][t]["drift"] for t in range(1, T)])
    assert np.sum(np.abs(gpu - emb)) < 0.1 * np.sum(np.abs(gpu - other))


@pytest.mark.parametrize("kind,n", [("mlp3", 81), ("flux6", 449), ("wan6", 785)])
def test_load_gate_closed_form_schedules(kind, n, lib):
    """A loaded gate with zero weights has z = its output bias: z = +1 always computes
    (front-loaded schedule), z = -1 always reuses (forced tail only)."""
    cfg = configs.get_config("tiny_ragged", gate_kind=kind)
    T, B = cfg["T"], 3
    ctx = bag.create(cfg, T=T, B=B)
    with pytest.raises(bag.BagError) as ei:
        ctx.load_gate(np.zeros(n + 1, np.float32))
    assert ei.value.status == 1
    for b_out, want in ((1.0, [1] * B + [0] * (T - B)), (-1.0, [1] + [0] * (T - B) + [1] * (B - 1))):
        theta = np.zeros(n, np.float32)
        theta[-1] = b_out
        ctx.load_gate(theta)
        _, _, m, log, nfe = _gpu_sample(cfg, T, B, ctx=ctx)
        assert list(m) == want and nfe == B
        assert np.all(log[1:, 3] == np.float32(b_out))
    ctx.close()


@pytest.mark.parametrize("name", ["tiny_ragged", "flux_small"])
def test_static_and_threshold_policies(name, lib):
    """Sec. 3.1's other two paradigms on the same path: the static evenly spaced schedule
    and the online threshold rule (schedule bit-exact on the GPU's logged drift)."""
    cfg = configs.get_config(name)
    T, B = cfg["T"], cfg["budgets"][0]
    W, g = synth.make_weights(cfg), synth.make_gate(cfg["gate_seed"])
    inp, got, m, log, nfe = _gpu_sample(cfg, T, B, policy=bag.POLICY_STATIC_UNIFORM)
    assert list(m) == O.static_uniform_schedule(B, T) and nfe == B
    ref = O.sample(cfg, W, g, inp, T=T, B=B, policy="uniform")
    rms = float(np.sqrt(np.mean(ref["x"] ** 2)))
    assert float(np.max(np.abs(got - ref["x"]))) <= TOL[cfg["dtype"]] * rms
    # a threshold between the smallest and largest drift of the run above
    d = np.sort(log[1:, 2])
    delta = float(d[len(d) // 2])
    inp, got, m, log, nfe = _gpu_sample(cfg, T, B, policy=bag.POLICY_THRESHOLD, delta=delta)
    want = [1] + [O.threshold_decision(float(log[t, 2]), delta) for t in range(1, T)]
    assert list(m) == want and nfe == sum(want)
    ref = O.sample(cfg, W, g, inp, T=T, B=B, policy=("threshold", delta),
                   drift_override=_gate_inputs(log))
    assert ref["mask"] == want
    rms = float(np.sqrt(np.mean(ref["x"] ** 2)))
    assert float(np.max(np.abs(got - ref["x"]))) <= TOL[cfg["dtype"]] * rms


# ---------------------------------------------------------------------------
# classifier-free guidance with one shared mask (App. A.1)
# ---------------------------------------------------------------------------
def _dev_uncond(cfg, inp):
    txt_u = torch.from_numpy(inp["txt_u"]).cuda()
    if cfg["dtype"] == "bf16":
        txt_u = txt_u.to(torch.bfloat16)
    return txt_u, torch.from_numpy(inp["pooled_u"]).cuda()


def _gpu_guided(cfg, T, B, inp):
    ctx = bag.create(cfg, T=T, B=B)
    x, txt, pooled = _dev_inputs(cfg, inp)
    txt_u, pooled_u = _dev_uncond(cfg, inp)
    ctx.reset()
    m, log, nfe = ctx.run(x, txt, pooled, txt_u, pooled_u)
    torch.cuda.synchronize()
    return ctx, x.cpu().numpy(), m, log, nfe


@pytest.mark.parametrize("name", ["tiny", "flux_small", "qwen_small", "wan_small"])
def test_guided_sample_parity(name, lib):
    """Both branches under one mask, signal on the conditional branch, v = v_u + g (v_c - v_u):
    schedule bit-exact on the GPU's gate inputs, latent within the dtype's bar; the host
    entry point gives the same bits as the device one."""
    g_scale = 4.0
    cfg = configs.get_config(name, guidance=g_scale)
    T, B = cfg["T"], cfg["budgets"][0]
    inp = synth.make_inputs(cfg)
    ctx, got, mask, log, nfe = _gpu_guided(cfg, T, B, inp)
    assert nfe == B and int(mask.sum()) == B and mask[0] == 1
    ctx.reset()
    xh = inp["x"].astype(np.float32).copy()
    mh, _, _ = ctx.run_host(xh, inp["txt"], inp["pooled"], inp["txt_u"], inp["pooled_u"])
    ctx.close()
    assert list(mh) == list(mask) and np.array_equal(xh, got)
    W, g = synth.make_weights(cfg), synth.make_gate(cfg["gate_seed"])
    ref = O.sample(cfg, W, g, inp, T=T, B=B, drift_override=_gate_inputs(log), guidance=g_scale)
    assert list(mask) == ref["mask"]
    rms = float(np.sqrt(np.mean(ref["x"] ** 2)))
    err = float(np.max(np.abs(got.astype(np.float64) - ref["x"])))
    assert err <= TOL[cfg["dtype"]] * rms, (err, rms)
    # guidance changed the result (the unconditional branch is not ignored)
    plain = O.sample(cfg, W, g, inp, T=T, B=B, policy=ref["mask"])
    assert float(np.max(np.abs(plain["x"] - ref["x"]))) > 10 * err


@pytest.mark.parametrize("name", ["tiny", "flux_small", "wan_small"])
def test_guided_identical_branches_equal_unguided(name, lib):
    """With the unconditional inputs equal to the conditional ones, v_u = v_c bit for bit,
    so any guidance scale reproduces the unguided sample exactly."""
    cfg = configs.get_config(name)
    T, B = cfg["T"], cfg["budgets"][0]
    inp, plain, m0, _, _ = _gpu_sample(cfg, T, B)
    same = dict(inp, txt_u=inp["txt"], pooled_u=inp["pooled"])
    ctx, got, m1, _, nfe = _gpu_guided(configs.get_config(name, guidance=7.5), T, B, same)
    ctx.close()
    assert list(m1) == list(m0) and nfe == B
    assert np.array_equal(got, plain)


@pytest.mark.parametrize("name", ["flux_small", "wan_small"])
def test_guided_budget_T_is_uncached_guided_sampling_bit_exact(name, lib):
    """B = T under guidance computes every step for both branches (the batch-2 stack) and
    equals the all-full policy bit for bit."""
    cfg = configs.get_config(name, guidance=3.0)
    T = 5
    inp = synth.make_inputs(cfg)
    ctx, a, ma, _, na = _gpu_guided(cfg, T, T, inp)
    ctx.close()
    ctx = bag.create(cfg, T=T, B=1)
    ctx.set_policy(bag.POLICY_FULL)
    x, txt, pooled = _dev_inputs(cfg, inp)
    txt_u, pooled_u = _dev_uncond(cfg, inp)
    ctx.reset()
    mb, _, nb = ctx.run(x, txt, pooled, txt_u, pooled_u)
    torch.cuda.synchronize()
    ctx.close()
    assert list(ma) == list(mb) == [1] * T and na == nb == T
    assert np.array_equal(a, x.cpu().numpy())


@pytest.mark.parametrize("name", ["flux_small", "wan_small"])
def test_guided_step_api_matches_run(name, lib):
    """bag_step under guidance (the batch-2 stack, one shared mask) reproduces bag_run bit
    for bit, step by step."""
    cfg = configs.get_config(name, guidance=2.5)
    T, B = 6, 3
    ctx = bag.create(cfg, T=T, B=B)
    inp = synth.make_inputs(cfg)
    x, txt, pooled = _dev_inputs(cfg, inp)
    txt_u, pooled_u = _dev_uncond(cfg, inp)
    x0 = x.clone()
    m_run, _, _ = ctx.run(x, txt, pooled, txt_u, pooled_u)
    ctx.reset()
    xs = x0.clone()
    flags = torch.zeros(T, dtype=torch.int32, device="cuda")
    for t in range(T):
        ctx.step(xs, t, txt, pooled, xs, flags[t:], txt_u, pooled_u)
    torch.cuda.synchronize()
    ctx.close()
    assert list(flags.cpu().numpy()) == list(m_run) and int(flags.sum()) == B
    assert torch.equal(xs, x)


def test_guided_context_requires_unconditional_inputs(lib):
    cfg = configs.get_config("tiny", guidance=2.0)
    ctx = bag.create(cfg, T=4, B=2)
    inp = synth.make_inputs(cfg)
    x, txt, pooled = _dev_inputs(cfg, inp)
    with pytest.raises(bag.BagError) as ei:
        ctx.run(x, txt, pooled)
    assert ei.value.status == 1
    ctx.close()


# ---------------------------------------------------------------------------
# QK-RMSNorm (FLUX / Qwen-Image blocks): fused into the QKV GEMM epilogue
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("name", ["single_small", "flux_small", "qwen_small"])
def test_qk_norm_sample_parity(name, lib):
    cfg = configs.get_config(name, qk_norm=True)
    T, B = cfg["T"], cfg["budgets"][0]
    ctx = bag.create(cfg, T=T, B=B)
    W = synth.make_weights(cfg)
    for blk in (0, len(W["blocks"]) - 1):
        for n in [k for k in W["blocks"][blk] if k.endswith("_norm")]:
            ref = W["blocks"][blk][n]
            assert np.array_equal(ctx.get_weight(blk, n, ref.size), ref), (blk, n)
    inp, got, mask, log, nfe = _gpu_sample(cfg, T, B, ctx=ctx)
    ctx.close()
    assert nfe == B and int(mask.sum()) == B
    g = synth.make_gate(cfg["gate_seed"])
    ref = O.sample(cfg, W, g, inp, T=T, B=B, drift_override=_gate_inputs(log))
    assert list(mask) == ref["mask"]
    rms = float(np.sqrt(np.mean(ref["x"] ** 2)))
    err = float(np.max(np.abs(got.astype(np.float64) - ref["x"])))
    assert err <= TOL[cfg["dtype"]] * rms, (err, rms)
    # the norm changed the result (the scales are not ignored)
    plain = O.sample(configs.get_config(name), synth.make_weights(configs.get_config(name)), g, inp,
                     T=T, B=B, policy=ref["mask"])
    assert float(np.max(np.abs(plain["x"] - ref["x"]))) > 10 * err


# ---------------------------------------------------------------------------
# samplers: UniPC (order 2 + corrector) and the time-shifted grid
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("name,over", [("tiny", dict(sampler="unipc", shift=3.0)),
                                       ("flux_small", dict(sampler="unipc")),
                                       ("wan_small", dict(sampler="euler", shift=5.0))],
                         ids=["tiny-unipc", "flux_small-unipc", "wan_small-euler-shift"])
def test_sampler_variant_parity(name, over, lib):
    cfg = configs.get_config(name, **over)
    T, B = cfg["T"], cfg["budgets"][0]
    inp, got, mask, log, nfe = _gpu_sample(cfg, T, B)
    assert nfe == B and int(mask.sum()) == B
    W, g = synth.make_weights(cfg), synth.make_gate(cfg["gate_seed"])
    ref = O.sample(cfg, W, g, inp, T=T, B=B, drift_override=_gate_inputs(log))
    assert list(mask) == ref["mask"]
    rms = float(np.sqrt(np.mean(ref["x"] ** 2)))
    err = float(np.max(np.abs(got.astype(np.float64) - ref["x"])))
    assert err <= TOL[cfg["dtype"]] * rms, (err, rms)


def test_unipc_budget_T_bit_exact_and_step_api(lib):
    """UniPC keeps its multistep history in the context: B = T equals uncached sampling
    bit for bit, and bag_step reproduces bag_run."""
    cfg = configs.get_config("wan_small")
    assert cfg["sampler"] == "unipc"
    T = 6
    _, a, ma, _, _ = _gpu_sample(cfg, T, T)
    _, b, mb, _, _ = _gpu_sample(cfg, T, 1, policy=bag.POLICY_FULL)
    assert list(ma) == list(mb) == [1] * T and np.array_equal(a, b)
    ctx = bag.create(cfg, T=T, B=3)
    inp = synth.make_inputs(cfg)
    x, txt, pooled = _dev_inputs(cfg, inp)
    x0 = x.clone()
    m_run, _, _ = ctx.run(x, txt, pooled)
    ctx.reset()
    xs = x0.clone()
    for t in range(T):
        ctx.step(xs, t, txt, pooled, xs)
    torch.cuda.synchronize()
    assert torch.equal(xs, x)
    ctx.close()


# ---------------------------------------------------------------------------
# failure path: a bounded wait that runs out is reported, sticky, and cleared by reset
# ---------------------------------------------------------------------------
def test_bounded_wait_timeout_is_reported_and_sticky(lib):
    import time
    cfg = configs.get_config("tiny")
    ctx = bag.create(cfg, T=4, B=2)
    t0 = time.time()
    st = ctx.check_wait_timeout()
    dt = time.time() - t0
    assert st == 5 and 1.0 < dt < 60.0, (st, dt)
    assert "bounded wait" in lib.bag_last_error(ctx.h).decode()
    inp = synth.make_inputs(cfg)
    x, txt, pooled = _dev_inputs(cfg, inp)
    with pytest.raises(bag.BagError) as ei:
        ctx.run(x, txt, pooled)
    assert ei.value.status == 5          # sticky until bag_reset
    ctx.reset()
    x, txt, pooled = _dev_inputs(cfg, inp)
    m, _, nfe = ctx.run(x, txt, pooled)  # the context is usable again
    torch.cuda.synchronize()
    assert nfe == 2 and int(m.sum()) == 2
    ctx.close()


# ---------------------------------------------------------------------------
# the extensions together: guidance + QK-norm + UniPC + a six-input gate
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("name,over", [
    ("flux_small", dict(guidance=3.0, qk_norm=True, sampler="unipc", shift=3.0, gate_kind="flux6")),
    ("qwen_small", dict(guidance=4.0, qk_norm=True, gate_kind="wan6")),
    ("wan_small", dict(guidance=5.0, gate_kind="wan6")),
], ids=["flux_small-all", "qwen_small-cfg-qkn", "wan_small-cfg-unipc"])
def test_extensions_combined_parity(name, over, lib):
    cfg = configs.get_config(name, **over)
    T, B = cfg["T"], cfg["budgets"][0]
    inp = synth.make_inputs(cfg)
    ctx, got, mask, log, nfe = _gpu_guided(cfg, T, B, inp)
    ctx.close()
    assert nfe == B and int(mask.sum()) == B and mask[0] == 1
    W = synth.make_weights(cfg)
    g = synth.make_gate_any(cfg["gate_seed"], cfg["gate_kind"])
    steps = [None] + [float(v) for v in log[1:, 13]]
    ref = O.sample(cfg, W, g, inp, T=T, B=B, drift_override=_gate_inputs(log),
                   step_override=steps, guidance=cfg["guidance"])
    assert list(mask) == ref["mask"]
    rms = float(np.sqrt(np.mean(ref["x"] ** 2)))
    err = float(np.max(np.abs(got.astype(np.float64) - ref["x"])))
    assert err <= TOL[cfg["dtype"]] * rms, (err, rms)


def test_set_budget_between_samples(lib):
    """bag_set_budget: the next sample spends exactly the new budget under Algorithm 2,
    and a static evenly spaced schedule is recomputed for it."""
    cfg = configs.get_config("tiny_ragged")
    T = cfg["T"]
    ctx = bag.create(cfg, T=T, B=2)
    for B in (2, 5, 1, T):
        ctx.set_budget(B)
        _, _, m, _, nfe = _gpu_sample(cfg, T, B, ctx=ctx)
        assert nfe == B and int(m.sum()) == B and m[0] == 1
    ctx.set_policy(bag.POLICY_STATIC_UNIFORM)
    for B in (3, 4):
        ctx.set_budget(B)
        _, _, m, _, nfe = _gpu_sample(cfg, T, B, ctx=ctx)
        assert list(m) == O.static_uniform_schedule(B, T) and nfe == B
    with pytest.raises(bag.BagError) as ei:
        ctx.set_budget(T + 1)
    assert ei.value.status == 1
    ctx.close()


@pytest.mark.parametrize("name", ["flux_small", "wan_small"])
def test_programmatic_launch_matches_stream_order(name, lib, monkeypatch):
    """Programmatic dependent launch changes only when each kernel's CTAs are scheduled,
    never what they compute: a sample with it (the default) and one with every kernel
    in plain stream order give the same latent and schedule bit for bit."""
    cfg = configs.get_config(name)
    T, B = 6, 3
    _, a, ma, la, na = _gpu_sample(cfg, T, B)
    monkeypatch.setenv("BAG_PDL", "0")
    _, b, mb, lb, nb = _gpu_sample(cfg, T, B)
    assert na == nb == B and list(ma) == list(mb)
    assert np.array_equal(a, b) and np.array_equal(la, lb)
