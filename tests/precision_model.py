"""Error model of the operand precision the bf16 backbones compute with (test helper).

The CUDA path of a bf16 configuration keeps the residual stream, LayerNorm statistics,
modulation vectors (the conditioning chain runs in split precision), the cached residual
and the latent in fp32, and rounds only the operands of its products:

  * every activation entering a projection (LayerNorm-modulated rows, the attention
    output, the GELU output, the final LayerNorm-modulated rows) to bf16, against
    bf16-valued weights; the latent enters the patch embedding as bf16 hi + lo halves,
    i.e. without that rounding;
  * the text tokens, which a bf16 context receives in bf16;
  * q, k and v (after QK-norm and RoPE) and the softmax probabilities P to fp16.

`operand_rounding(O)` evaluates the fp64 oracle's own functions with exactly these
roundings inserted and everything else in float64.  The difference between its result
and the plain oracle is the error that this precision carries by itself, whatever
kernel computes it; tests bound the GPU's error by a small multiple of it.  It imports
only the oracle and the seeded generator's rounding helper, never the CUDA path.
"""

import contextlib
import math

import numpy as np

from paper_2608_09231_gb300 import synth


def to_bf16(x):
    return synth.bf16_round(np.asarray(x, np.float32)).astype(np.float64)


def to_f16(x):
    return np.asarray(x, np.float64).astype(np.float16).astype(np.float64)


@contextlib.contextmanager
def operand_rounding(O):
    """Within the block, the oracle module O computes with the operand roundings above."""
    lin, att, cond, bmod, fin = O.linear, O.attention, O.conditioning, O.block_modulation, O.final_layer
    pe = O.patch_embed

    def linear(x, w, b=None):
        return lin(to_bf16(x), w, b)

    def attention(q, k, v, q_rows=None):
        q, k, v = to_f16(q), to_f16(k), to_f16(v)
        if q_rows is not None:
            q = q[q_rows]
        out = np.empty(q.shape, dtype=np.float64)
        for h in range(q.shape[1]):
            s = q[:, h, :] @ k[:, h, :].T / math.sqrt(q.shape[-1])
            e = np.exp(s - s.max(axis=-1, keepdims=True))
            out[:, h, :] = (to_f16(e) @ v[:, h, :]) / e.sum(axis=-1, keepdims=True)
        return out

    def exact(fn):
        def run(*a, **k):
            O.linear = lin
            try:
                return fn(*a, **k)
            finally:
                O.linear = linear
        return run

    def final_layer(G, vec, h_img):
        d = h_img.shape[1]
        mod = lin(O.silu(vec), G["fmod_w"], G["fmod_b"])
        return lin(to_bf16(O.modulate(O.layer_norm(h_img), mod[:d], mod[d:])), G["fin_w"], G["fin_b"])

    O.linear, O.attention, O.final_layer = linear, attention, final_layer
    O.conditioning, O.block_modulation, O.patch_embed = exact(cond), exact(bmod), exact(pe)
    try:
        yield
    finally:
        O.linear, O.attention, O.conditioning, O.block_modulation, O.final_layer = lin, att, cond, bmod, fin
        O.patch_embed = pe


def bf16_inputs(inp):
    """The inputs as a bf16 context receives them: text tokens (both branches) in bf16."""
    out = dict(inp)
    for k in ("txt", "txt_u"):
        if k in out:
            out[k] = to_bf16(out[k])
    return out
