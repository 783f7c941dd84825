"""The operand-precision error model (tests/precision_model.py) rounds exactly where it
says and nowhere else, and leaves the oracle untouched outside its block."""

import math

import numpy as np

from oracle import bag_oracle as O
from paper_2608_09231_gb300 import configs, synth
from precision_model import bf16_inputs, operand_rounding, to_bf16, to_f16


def test_roundings_and_restore():
    rng = np.random.default_rng(3)
    x, w, b = rng.normal(size=(5, 16)), to_bf16(rng.normal(size=(8, 16))), rng.normal(size=8)
    q, k, v = rng.normal(size=(6, 2, 8)), rng.normal(size=(7, 2, 8)), rng.normal(size=(7, 2, 8))
    lin, att, pe = O.linear, O.attention, O.patch_embed
    G = {"pe_w": w, "pe_b": b}
    with operand_rounding(O):
        assert np.array_equal(O.linear(x, w, b), lin(to_bf16(x), w, b))
        assert np.array_equal(O.patch_embed(G, x), lin(x, w, b))  # split-precision latent
        got = O.attention(q, k, v, q_rows=np.array([1, 4]))
    assert O.linear is lin and O.attention is att and O.patch_embed is pe
    qf, kf, vf = to_f16(q), to_f16(k), to_f16(v)
    for r, qi in enumerate([1, 4]):
        for h in range(2):
            s = np.array([qf[qi, h] @ kf[j, h] for j in range(7)]) / math.sqrt(8)
            e = np.exp(s - s.max())
            want = (to_f16(e) @ vf[:, h]) / e.sum()
            assert np.allclose(got[r, h], want, rtol=1e-12, atol=1e-12)
    # bf16 keeps 8 significant bits, fp16 11: the rounding errors differ by about 2^3
    z = rng.normal(size=10000)
    e16, eb = np.sqrt(np.mean((to_f16(z) - z) ** 2)), np.sqrt(np.mean((to_bf16(z) - z) ** 2))
    assert 6 < eb / e16 < 10


def test_conditioning_stays_exact_and_block_error_is_small():
    """The conditioning chain (split precision on the GPU) is not rounded; a tiny
    single-stream block under the model differs from the oracle by a relative error of
    the order of bf16 rounding."""
    cfg = configs.get_config("single_small")
    W = synth.make_weights(cfg, blocks=[0])
    inp = bf16_inputs(synth.make_inputs(cfg))
    G = O.to64(W)["global"]
    vec = O.conditioning(cfg, G, 0.6, inp["pooled"].astype(np.float64))
    with operand_rounding(O):
        assert np.array_equal(O.conditioning(cfg, G, 0.6, inp["pooled"].astype(np.float64)), vec)
        N, d = cfg["n_img"] + cfg["n_txt"], cfg["hidden"]
        h = synth.normal(5, 900, N * d, 1.0).reshape(N, d).astype(np.float64)
        m = O.forward_block(cfg, W, 0, h, vec)
    ref = O.forward_block(cfg, W, 0, h, vec)
    rel = np.sqrt(np.mean((m - ref) ** 2)) / np.sqrt(np.mean((ref - h) ** 2))
    assert 1e-4 < rel < 2e-2, rel
