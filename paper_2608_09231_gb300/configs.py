"""Architecture and sampling configurations (shapes only, no arithmetic).

The paper runs its gate on FLUX.1-dev, Qwen-Image and Wan2.1 backbones (Sec. 4.1) and
states the problem as T sequential compute-or-reuse decisions under an NFE budget B
(Sec. 3.1, Algorithm 2).  The paper never lists the backbones' internals; the shapes
below are the public FLUX-, Qwen-Image- and Wan2.1-14B-sized layouts of the workloads
the method is evaluated on, plus a tiny fp32 stack for exhaustive parity and reduced
("small") variants that the fp64 oracle finishes in seconds.

Every field is plain data shared by the CUDA path's binding, the tests and the oracle.

Fields
------
kind        'single' (single-stream blocks only), 'mmdit' (double-stream then
            single-stream blocks: FLUX/Qwen), 'wan' (self-attn + cross-attn + FFN blocks)
hidden      model width d
heads       attention heads H (head_dim = hidden // heads)
mlp         MLP width F
n_double    number of double-stream blocks ('mmdit')
n_single    number of single-stream blocks ('single', 'mmdit')
n_wan       number of Wan blocks ('wan')
grid        (frames, rows, cols) of image tokens; n_img = product
n_txt       text tokens (joint attention) or context tokens (Wan cross-attention)
patch_ch    channels per image token in the latent (64 = 16-ch latent x 2x2 patch)
rope_axes   head-dim split of the rotary embedding over the (frame, row, col) axes
dtype       'f32' or 'bf16' (GEMM / attention operand type)
gate_kind   'mlp3' (3 inputs, default), 'flux6' or 'wan6' (the paper's six-input gates)
observable  what the trajectory signal reads: 'modulated' (default; the first block's
            modulated image-stream input) or 'embedded' (the post-patch-embedding
            tokens, the paper's observable)
"""

import copy

TEMB_DIM = 256          # sinusoidal timestep-embedding width (FLUX/Wan convention)
ROPE_THETA = 10000.0
LN_EPS = 1e-6

_BASE = {
    # tiny stack (2 single-stream blocks, d 256): fp32 end to end, exhaustive parity
    "tiny": dict(kind="single", hidden=256, heads=4, mlp=1024, n_double=0, n_single=2,
                 n_wan=0, grid=(1, 16, 16), n_txt=32, patch_ch=64, rope_axes=(0, 32, 32),
                 dtype="f32", weight_seed=0, gate_seed=100, T=10, budgets=(5,)),
    # one FLUX-shaped single-stream block (block forward + skip-path kernels only)
    "flux_block": dict(kind="single", hidden=3072, heads=24, mlp=12288, n_double=0,
                       n_single=1, n_wan=0, grid=(1, 64, 64), n_txt=512, patch_ch=64,
                       rope_axes=(16, 56, 56), dtype="bf16", weight_seed=1, gate_seed=101,
                       T=50, budgets=(25,)),
    # FLUX.1-dev-shaped MMDiT at 1024x1024
    "flux": dict(kind="mmdit", hidden=3072, heads=24, mlp=12288, n_double=19, n_single=38,
                 n_wan=0, grid=(1, 64, 64), n_txt=512, patch_ch=64, rope_axes=(16, 56, 56),
                 dtype="bf16", weight_seed=2, gate_seed=102, T=50, budgets=(25, 20, 15, 10)),
    # Qwen-Image-shaped MMDiT at 1328x1328 (83 x 83 tokens)
    "qwen": dict(kind="mmdit", hidden=3072, heads=24, mlp=12288, n_double=60, n_single=0,
                 n_wan=0, grid=(1, 83, 83), n_txt=256, patch_ch=64, rope_axes=(16, 56, 56),
                 dtype="bf16", weight_seed=3, gate_seed=103, T=50, budgets=(20, 10)),
    # Wan2.1-14B-shaped video DiT, 81 frames 480x832 -> 21 x 30 x 52 tokens; sampled with
    # UniPC as in the paper's Wan runs, on a time-shifted grid (shift 5)
    "wan": dict(kind="wan", hidden=5120, heads=40, mlp=13824, n_double=0, n_single=0,
                n_wan=40, grid=(21, 30, 52), n_txt=512, patch_ch=64, rope_axes=(44, 42, 42),
                dtype="bf16", weight_seed=4, gate_seed=104, T=50, budgets=(20,),
                sampler="unipc", shift=5.0),
}

# Reduced variants at which the fp64 oracle runs a whole sample in seconds.  Token
# counts are deliberately ragged (not multiples of the 128-row tiles).
_SMALL = {
    "flux_small": dict(_BASE["flux"], hidden=512, heads=4, mlp=2048, n_double=2, n_single=2,
                       grid=(1, 18, 21), n_txt=77, T=10, budgets=(5,)),
    "qwen_small": dict(_BASE["qwen"], hidden=512, heads=4, mlp=1536, n_double=3,
                       grid=(1, 17, 19), n_txt=40, T=10, budgets=(4,)),
    "wan_small": dict(_BASE["wan"], hidden=512, heads=4, mlp=1536, n_wan=2, grid=(3, 10, 13),
                      n_txt=70, rope_axes=(44, 42, 42), T=10, budgets=(4,)),
    "single_small": dict(_BASE["flux_block"], hidden=512, heads=4, mlp=2048, n_single=2,
                         grid=(1, 20, 23), n_txt=45, T=8, budgets=(3,)),
    "tiny_ragged": dict(_BASE["tiny"], grid=(1, 13, 11), n_txt=19, T=7, budgets=(3,)),
}

# Production width at reduced depth and token count: the blocks, head count, MLP width
# and RoPE layout of the FLUX-, Qwen-Image- and Wan2.1-14B-shaped stacks, with one or
# two blocks and 1000-1650 image tokens, so that the fp64 oracle runs a whole short
# sample while every stack projection has enough 256 x 256 tiles (at least one per CTA
# pair) to run on the CTA-pair GEMM.
_WIDE = {
    "flux_wide": dict(_BASE["flux"], n_double=1, n_single=1, grid=(1, 36, 36), n_txt=512,
                      T=6, budgets=(3,)),
    "qwen_wide": dict(_BASE["qwen"], n_double=1, grid=(1, 41, 40), n_txt=256, T=6,
                      budgets=(3,)),
    "wan_wide": dict(_BASE["wan"], n_wan=1, grid=(3, 16, 21), n_txt=512, T=6, budgets=(3,)),
}


def get_config(name, **overrides):
    """Return a fresh config dict with derived fields filled in."""
    if name in _BASE:
        cfg = copy.deepcopy(_BASE[name])
    elif name in _SMALL:
        cfg = copy.deepcopy(_SMALL[name])
    elif name in _WIDE:
        cfg = copy.deepcopy(_WIDE[name])
    else:
        raise KeyError(f"unknown config {name!r}")
    cfg.update(overrides)
    cfg.setdefault("gate_kind", "mlp3")
    cfg.setdefault("sampler", "euler")     # "euler" or "unipc"
    cfg.setdefault("shift", 1.0)           # time shift of the sigma grid
    cfg.setdefault("observable", "modulated")
    cfg["name"] = name
    d, h = cfg["hidden"], cfg["heads"]
    assert d % h == 0
    cfg["head_dim"] = d // h
    g = cfg["grid"]
    cfg["n_img"] = g[0] * g[1] * g[2]
    assert sum(cfg["rope_axes"]) == cfg["head_dim"], "RoPE axes must tile the head dim"
    for a in cfg["rope_axes"]:
        assert a % 2 == 0
    return cfg


def config_names():
    return list(_BASE) + list(_SMALL) + list(_WIDE)
