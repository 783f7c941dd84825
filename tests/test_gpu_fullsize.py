"""Full-size checks at the benchmark workloads' shapes, in the launch configuration the
benchmark times.

* One block of each kind (FLUX single-stream, FLUX and Qwen-Image double-stream,
  Wan2.1-14B) at full width and full token count, run through bag_forward_block,
  against the fp64 oracle evaluated one sampled row at a time (the oracle computes the
  keys and values of every token, and the block output only at the sampled rows).
  Tolerance, from the operand precision rather than from any kernel: a block output is
  h + g * o, and o passes through the roundings of its operands (bf16 projection inputs,
  fp16 q, k, v and P), each a relative error of at most 2^-8 (bf16) or 2^-11 (fp16), so
  the error scales with the element's own update |g * o|, which at full width reaches
  ~5x the output RMS in columns with large adaLN gates.  Bar per element:
  |err| <= 2e-2 x RMS(ref) + 2^-7 x |ref - h|.  Over the sampled rows the error model of
  tests/precision_model.py (the oracle evaluated with exactly those operand roundings)
  predicts RMS(err) for the block; the GPU's RMS(err) must stay within 1.25x of it, so
  the kernels add at most a quarter to the error their declared precision carries by
  itself.  The text tokens enter both sides in bf16, as a bf16 context receives them.
* Whole samples at full size: properties that hold at any size — realised NFE = B for
  every configured budget, m_0 = 1, the schedule equals Algorithm 2 applied to the gate
  bits the oracle computes from the GPU's logged gate inputs, and B = T reproduces
  uncached sampling bit for bit.
"""

import numpy as np
import pytest
import torch

from oracle import bag_oracle as O
from paper_2608_09231_gb300 import bag, configs, synth
from precision_model import bf16_inputs, operand_rounding

pytestmark = pytest.mark.gpu


def _dev(cfg, inp):
    txt = torch.from_numpy(inp["txt"]).cuda()
    if cfg["dtype"] == "bf16":
        txt = txt.to(torch.bfloat16)
    return txt, torch.from_numpy(inp["pooled"]).cuda()


BLOCKS = [
    ("flux_block", {}, [0, 1, 300, 511, 512, 513, 2100, 4607]),
    ("flux_block", dict(qk_norm=True), [0, 2, 511, 512, 2047, 4607]),
    ("flux", dict(n_double=1, n_single=0), [0, 255, 511, 512, 1000, 3333, 4607]),
    ("flux", dict(n_double=1, n_single=0, qk_norm=True), [1, 510, 513, 4000]),
    ("qwen", dict(n_double=1), [0, 255, 256, 257, 4000, 7144]),
    ("wan", dict(n_wan=1), [0, 1, 1559, 16000, 32759]),
]


@pytest.mark.parametrize("name,over,rows", BLOCKS,
                         ids=[b[0] + "-" + "-".join(sorted(b[1])) for b in BLOCKS])
def test_block_full_size_sampled_rows(name, over, rows, lib):
    cfg = configs.get_config(name, **over)
    d = cfg["hidden"]
    N = cfg["n_img"] + (0 if cfg["kind"] == "wan" else cfg["n_txt"])
    ctx = bag.create(cfg, T=cfg["T"], B=1)
    inp = synth.make_inputs(cfg)
    txt, pooled = _dev(cfg, inp)
    ctx.prepare(txt, pooled)
    h0 = synth.normal(cfg["weight_seed"], 900, N * d, 1.0).reshape(N, d)
    h = torch.from_numpy(h0).cuda()
    ctx.forward_block(0, 0, h)
    torch.cuda.synchronize()
    got = h.cpu().numpy()[rows].astype(np.float64)
    ctx.close()
    W = synth.make_weights(cfg, blocks=[0])
    G = O.to64(W)["global"]
    vec = O.conditioning(cfg, G, 1.0, inp["pooled"].astype(np.float64))
    txt = bf16_inputs(inp)["txt"]
    h64 = h0.astype(np.float64)
    ref = O.forward_block(cfg, W, 0, h64, vec, rows=np.array(rows), txt=txt)
    with operand_rounding(O):
        model = O.forward_block(cfg, W, 0, h64, vec, rows=np.array(rows), txt=txt)
    rms = float(np.sqrt(np.mean(ref ** 2)))
    upd = ref - h0[rows]
    err = np.abs(got - ref)
    rms_err, rms_model = float(np.sqrt(np.mean(err ** 2))), float(np.sqrt(np.mean((model - ref) ** 2)))
    rms_upd = float(np.sqrt(np.mean(upd ** 2)))
    print(f"{name} {over}: max|err| = {err.max():.4e} = {err.max() / rms:.3e} x RMS(ref) "
          f"(model {np.max(np.abs(model - ref)) / rms:.3e}); RMS(err) / RMS(update) = "
          f"{rms_err / rms_upd:.4e} (model {rms_model / rms_upd:.4e})")
    bar = 2e-2 * rms + 2.0 ** -7 * np.abs(upd)
    assert np.all(err <= bar), (float(err.max()), float((err / bar).max()))
    assert rms_err <= 1.25 * rms_model, (rms_err, rms_model)
    # the block changed the stream (it is not an identity pass)
    assert rms_upd > 100 * rms_err


def _sample(ctx, cfg, inp):
    x = torch.from_numpy(inp["x"].copy()).cuda()
    txt, pooled = _dev(cfg, inp)
    ctx.reset()
    m, log, nfe = ctx.run(x, txt, pooled)
    torch.cuda.synchronize()
    return x.cpu().numpy(), m, log, nfe


@pytest.mark.parametrize("name,T,budgets", [("flux", 50, (25, 20, 15, 10)), ("qwen", 50, (20, 10)),
                                            ("wan", 10, (3,))])
def test_full_size_schedules(name, T, budgets, lib):
    cfg = configs.get_config(name)
    inp = synth.make_inputs(cfg)
    g = synth.make_gate(cfg["gate_seed"])
    ctx = None
    for B in budgets:
        if ctx is not None:
            ctx.close()
        ctx = bag.create(cfg, T=T, B=B)
        x, m, log, nfe = _sample(ctx, cfg, inp)
        assert nfe == B and int(m.sum()) == B and m[0] == 1
        assert np.all(np.isfinite(x))
        bits = [None]
        for t in range(1, T):
            f = [np.float32(v) for v in log[t, 0:3]]
            z = O.gate_logit(f, g)
            assert z == np.float32(log[t, 3])
            bits.append(1 if z > O.gate_threshold(0.5) else 0)
        assert list(m) == O.schedule_from_gate_bits(bits, B, T)
    ctx.close()


def test_flux_full_size_budget_T_is_uncached(lib):
    cfg = configs.get_config("flux")
    inp = synth.make_inputs(cfg)
    T = 6
    ctx = bag.create(cfg, T=T, B=T)
    a, ma, _, _ = _sample(ctx, cfg, inp)
    ctx.set_policy(bag.POLICY_FULL)
    b, mb, _, _ = _sample(ctx, cfg, inp)
    ctx.close()
    assert list(ma) == list(mb) == [1] * T
    assert np.array_equal(a, b)


def test_full_size_guided_schedule(lib):
    """Qwen-Image-sized sample under classifier-free guidance (both branches, one mask):
    NFE = B, m_0 = 1, and the schedule is Algorithm 2 on the gate bits the oracle computes
    from the logged inputs of the conditional branch."""
    cfg = configs.get_config("qwen", guidance=4.0)
    T, B = 50, 10
    inp = synth.make_inputs(cfg)
    g = synth.make_gate(cfg["gate_seed"])
    ctx = bag.create(cfg, T=T, B=B)
    x = torch.from_numpy(inp["x"].copy()).cuda()
    txt, pooled = _dev(cfg, inp)
    txt_u = torch.from_numpy(inp["txt_u"]).cuda().to(torch.bfloat16)
    pooled_u = torch.from_numpy(inp["pooled_u"]).cuda()
    ctx.reset()
    m, log, nfe = ctx.run(x, txt, pooled, txt_u, pooled_u)
    torch.cuda.synchronize()
    ctx.close()
    assert nfe == B and int(m.sum()) == B and m[0] == 1
    assert np.all(np.isfinite(x.cpu().numpy()))
    bits = [None]
    for t in range(1, T):
        z = O.gate_logit([np.float32(v) for v in log[t, 0:3]], g)
        assert z == np.float32(log[t, 3])
        bits.append(1 if z > O.gate_threshold(0.5) else 0)
    assert list(m) == O.schedule_from_gate_bits(bits, B, T)
