"""Seeded synthetic inputs: one counter-based generator, host side (numpy).

This module holds none of the method's arithmetic.  It only turns (seed, tensor key,
element index) into numbers, so that the fp64 oracle and the CUDA path see the same
weights and inputs.  The CUDA library carries its own implementation of the same
generator (device kernel for the large weight tensors, host C++ for the gate); both are
written from the published definition of SplitMix64 (Steele, Lea and Flood, "Fast
splittable pseudorandom number generators", OOPSLA 2014):

    state_i = s + (i + 1) * 0x9E3779B97F4A7C15          (mod 2^64)
    out_i   = mix(state_i)
    mix(z)  : z ^= z >> 30; z *= 0xBF58476D1CE4E5B9;
              z ^= z >> 27; z *= 0x94D049BB133111EB; z ^= z >> 31

with the stream start  s = mix(seed * 0x9E3779B97F4A7C15 ^ mix(key)).

Distributions (all exactly reproducible in IEEE fp32 on any machine):
  normal(std)   Irwin-Hall sum of the four 16-bit chunks of out_i, centred:
                q = a+b+c+d - 131070 (an integer, exact in fp32), value = fp32(q) * c32
                with c32 = fp32(std * sqrt(3) / 65536), so the variance is std^2.
  uniform(lo,hi) u = fp32(out_i >> 40) * 2^-24; value = lo + (hi - lo) * u, each
                operation rounded separately in fp32.
bf16 storage uses round-to-nearest-even of the fp32 value.
"""

import concurrent.futures
import os

import numpy as np

from .configs import TEMB_DIM

GOLDEN = np.uint64(0x9E3779B97F4A7C15)
M1 = np.uint64(0xBF58476D1CE4E5B9)
M2 = np.uint64(0x94D049BB133111EB)


def _mix(z):
    z = np.asarray(z, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * M1
        z = (z ^ (z >> np.uint64(27))) * M2
    return z ^ (z >> np.uint64(31))


def stream_start(seed, key):
    with np.errstate(over="ignore"):
        a = np.uint64(seed) * GOLDEN
    return _mix(a ^ _mix(np.uint64(key)))


def raw_u64(seed, key, n, offset=0):
    s = stream_start(seed, key)
    idx = np.arange(offset + 1, offset + n + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        st = s + idx * GOLDEN
    return _mix(st)


def normal_scale(std):
    return np.float32(float(std) * np.sqrt(3.0) / 65536.0)


def _normal_range(out, s, c32, lo, hi, offset, chunk=1 << 16):
    """Fill out[lo:hi] (cache-sized chunks, in-place ufuncs: numpy releases the GIL)."""
    n = min(chunk, hi - lo)
    base = np.arange(1, n + 1, dtype=np.uint64) * GOLDEN
    z = np.empty(n, np.uint64)
    t = np.empty(n, np.uint64)
    q = np.empty(n, np.uint64)
    m = np.uint64(0xFFFF)
    with np.errstate(over="ignore"):
        for a in range(lo, hi, chunk):
            k = min(chunk, hi - a)
            zz, tt, qq = z[:k], t[:k], q[:k]
            np.add(base[:k], s + np.uint64(offset + a) * GOLDEN, out=zz)
            np.right_shift(zz, np.uint64(30), out=tt)
            np.bitwise_xor(zz, tt, out=zz)
            np.multiply(zz, M1, out=zz)
            np.right_shift(zz, np.uint64(27), out=tt)
            np.bitwise_xor(zz, tt, out=zz)
            np.multiply(zz, M2, out=zz)
            np.right_shift(zz, np.uint64(31), out=tt)
            np.bitwise_xor(zz, tt, out=zz)
            np.bitwise_and(zz, m, out=qq)
            for sh in (16, 32):
                np.right_shift(zz, np.uint64(sh), out=tt)
                np.bitwise_and(tt, m, out=tt)
                np.add(qq, tt, out=qq)
            np.right_shift(zz, np.uint64(48), out=tt)
            np.add(qq, tt, out=qq)
            o = out[a:a + k]
            o[:] = qq.view(np.int64) - 131070
            np.multiply(o, c32, out=o)


def normal(seed, key, n, std, offset=0):
    """n fp32 samples of the Irwin-Hall(4) normal approximation with the given std."""
    out = np.empty(n, dtype=np.float32)
    c32 = normal_scale(std)
    s = stream_start(seed, key)
    nt = min(16, os.cpu_count() or 1) if n >= (1 << 22) else 1
    if nt == 1:
        _normal_range(out, s, c32, 0, n, offset)
        return out
    step = -(-n // nt)
    with concurrent.futures.ThreadPoolExecutor(nt) as ex:
        list(ex.map(lambda i: _normal_range(out, s, c32, i * step, min(n, (i + 1) * step), offset),
                    range(nt)))
    return out


def uniform(seed, key, n, lo, hi):
    u = raw_u64(seed, key, n)
    f = (u >> np.uint64(40)).astype(np.float32) * np.float32(2.0 ** -24)
    return np.float32(lo) + (np.float32(hi) - np.float32(lo)) * f


def bf16_round(x):
    """Round fp32 values to the nearest bf16 (ties to even); returns fp32 values.
    (Finite inputs; the rounding carry may step into the exponent, as it should.)"""
    x = np.array(x, dtype=np.float32, copy=True, order="C")
    u = x.reshape(-1).view(np.uint32)
    step = 1 << 18

    def rnd(a):
        v = u[a:a + step]
        r = (v >> np.uint32(16)) & np.uint32(1)
        r += np.uint32(0x7FFF)
        v += r
        v &= np.uint32(0xFFFF0000)

    starts = range(0, u.size, step)
    if u.size >= (1 << 22):
        with concurrent.futures.ThreadPoolExecutor(min(16, os.cpu_count() or 1)) as ex:
            list(ex.map(rnd, starts))
    else:
        for a in starts:
            rnd(a)
    return x


def bf16_bits(x):
    """Bit pattern (uint16) of fp32 values that are already bf16-representable."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    return (x.view(np.uint32) >> np.uint32(16)).astype(np.uint16)


# ---------------------------------------------------------------------------
# Tensor inventory.  key = block_slot * 256 + tensor_id; block_slot 0 holds the global
# tensors, slot 1 + i the i-th block in execution order (double blocks, then single).
# Weights are [out, in] row-major (out features x in features).
# ---------------------------------------------------------------------------
WEIGHT_STD = 0.02
BIAS_STD = 0.02

GLOBAL_IDS = {
    "pe_w": 0, "pe_b": 1, "t1_w": 2, "t1_b": 3, "t2_w": 4, "t2_b": 5,
    "fmod_w": 6, "fmod_b": 7, "fin_w": 8, "fin_b": 9, "tproj_w": 10, "tproj_b": 11,
}
SINGLE_IDS = {"mod_w": 0, "mod_b": 1, "lin1_w": 2, "lin1_b": 3, "lin2_w": 4, "lin2_b": 5,
              "q_norm": 6, "k_norm": 7}
DOUBLE_IDS = {}
for _i, _s in enumerate(("img", "txt")):
    for _j, _n in enumerate(("mod", "qkv", "proj", "up", "down")):
        DOUBLE_IDS[f"{_s}_{_n}_w"] = _i * 10 + 2 * _j
        DOUBLE_IDS[f"{_s}_{_n}_b"] = _i * 10 + 2 * _j + 1
    DOUBLE_IDS[f"{_s}_q_norm"] = 20 + 2 * _i
    DOUBLE_IDS[f"{_s}_k_norm"] = 21 + 2 * _i
# QK-norm scales (optional, cfg["qk_norm"]): 1 + N(0, NORM_STD) per head channel.
NORM_STD = 0.02
WAN_IDS = {"mod_tab": 0, "sa_qkv_w": 1, "sa_qkv_b": 2, "sa_o_w": 3, "sa_o_b": 4,
           "ca_q_w": 5, "ca_q_b": 6, "ca_kv_w": 7, "ca_kv_b": 8, "ca_o_w": 9, "ca_o_b": 10,
           "ffn_up_w": 11, "ffn_up_b": 12, "ffn_down_w": 13, "ffn_down_b": 14}


def global_shapes(cfg):
    d, C = cfg["hidden"], cfg["patch_ch"]
    s = {"pe_w": (d, C), "pe_b": (d,), "t1_w": (d, TEMB_DIM), "t1_b": (d,),
         "t2_w": (d, d), "t2_b": (d,), "fmod_w": (2 * d, d), "fmod_b": (2 * d,),
         "fin_w": (C, d), "fin_b": (C,)}
    if cfg["kind"] == "wan":
        s["tproj_w"] = (6 * d, d)
        s["tproj_b"] = (6 * d,)
    return s


def block_shapes(cfg, btype):
    d, F = cfg["hidden"], cfg["mlp"]
    qkn = bool(cfg.get("qk_norm"))
    dh = d // cfg["heads"] if qkn else 0
    if btype == "single":
        s = {"mod_w": (3 * d, d), "mod_b": (3 * d,), "lin1_w": (3 * d + F, d),
             "lin1_b": (3 * d + F,), "lin2_w": (d, d + F), "lin2_b": (d,)}
        if qkn:
            s.update({"q_norm": (dh,), "k_norm": (dh,)})
        return s
    if btype == "double":
        s = {}
        for st in ("img", "txt"):
            s.update({f"{st}_mod_w": (6 * d, d), f"{st}_mod_b": (6 * d,),
                      f"{st}_qkv_w": (3 * d, d), f"{st}_qkv_b": (3 * d,),
                      f"{st}_proj_w": (d, d), f"{st}_proj_b": (d,),
                      f"{st}_up_w": (F, d), f"{st}_up_b": (F,),
                      f"{st}_down_w": (d, F), f"{st}_down_b": (d,)})
            if qkn:
                s.update({f"{st}_q_norm": (dh,), f"{st}_k_norm": (dh,)})
        return s
    if btype == "wan":
        if qkn:
            raise ValueError("QK-norm is built for single- and double-stream blocks only")
        return {"mod_tab": (6 * d,), "sa_qkv_w": (3 * d, d), "sa_qkv_b": (3 * d,),
                "sa_o_w": (d, d), "sa_o_b": (d,), "ca_q_w": (d, d), "ca_q_b": (d,),
                "ca_kv_w": (2 * d, d), "ca_kv_b": (2 * d,), "ca_o_w": (d, d), "ca_o_b": (d,),
                "ffn_up_w": (F, d), "ffn_up_b": (F,), "ffn_down_w": (d, F),
                "ffn_down_b": (d,)}
    raise ValueError(btype)


def block_types(cfg):
    """Block types in execution order."""
    if cfg["kind"] == "wan":
        return ["wan"] * cfg["n_wan"]
    return ["double"] * cfg["n_double"] + ["single"] * cfg["n_single"]


def _ids(btype):
    return {"single": SINGLE_IDS, "double": DOUBLE_IDS, "wan": WAN_IDS}[btype]


def _gen(cfg, slot, tid, name, shape):
    n = int(np.prod(shape))
    if name.endswith("_norm"):
        return np.float32(1.0) + normal(cfg["weight_seed"], slot * 256 + tid, n, NORM_STD).reshape(shape)
    std = BIAS_STD if (name.endswith("_b") or name == "mod_tab") else WEIGHT_STD
    v = normal(cfg["weight_seed"], slot * 256 + tid, n, std).reshape(shape)
    # matrices are stored in the GEMM operand type; biases/tables stay fp32
    if cfg["dtype"] == "bf16" and len(shape) == 2:
        v = bf16_round(v)
    return v


def make_weights(cfg, blocks=None):
    """All weights as fp32 numpy arrays (bf16-valued for bf16 configs).

    blocks: optional list of block indices to generate (others are None), so that a
    reduced-depth oracle run can fetch exactly the blocks it needs."""
    out = {"global": {}, "blocks": []}
    for name, shape in global_shapes(cfg).items():
        out["global"][name] = _gen(cfg, 0, GLOBAL_IDS[name], name, shape)
    for i, bt in enumerate(block_types(cfg)):
        if blocks is not None and i not in blocks:
            out["blocks"].append(None)
            continue
        ids = _ids(bt)
        out["blocks"].append({"type": bt, **{n: _gen(cfg, 1 + i, ids[n], n, s)
                                             for n, s in block_shapes(cfg, bt).items()}})
    return out


# Gate parameters: MLP 3 -> 16 -> 1 with Xavier-uniform bounds, drawn on the host.
GATE_IN, GATE_HID = 3, 16
GATE_KEYS = {"w1": 1, "b1": 2, "w2": 3, "b2": 4}


def make_gate(gate_seed):
    """Seeded gate parameters (fp32): w1 [16,3], b1 [16], w2 [16], b2 [1], mu [3], sd [3]."""
    a1 = float(np.sqrt(6.0 / (GATE_IN + GATE_HID)))
    a2 = float(np.sqrt(6.0 / (GATE_HID + 1)))
    g = {
        "w1": uniform(gate_seed, GATE_KEYS["w1"], GATE_HID * GATE_IN, -a1, a1).reshape(GATE_HID, GATE_IN),
        "b1": uniform(gate_seed, GATE_KEYS["b1"], GATE_HID, -0.1, 0.1),
        "w2": uniform(gate_seed, GATE_KEYS["w2"], GATE_HID, -a2, a2),
        "b2": uniform(gate_seed, GATE_KEYS["b2"], 1, -0.1, 0.1),
        "mu": np.zeros(GATE_IN, np.float32),
        "sd": np.ones(GATE_IN, np.float32),
    }
    return g


def gate_flat(g):
    """Flat parameter vector: for the 3-input gate w1 (row-major), b1, w2, b2 (81 floats);
    for the 6-input gates every layer's W [out, in] (row-major) then b, in layer order."""
    if g.get("kind", "mlp3") == "mlp3":
        return np.concatenate([g["w1"].ravel(), g["b1"], g["w2"], g["b2"]]).astype(np.float32)
    return np.concatenate([np.concatenate([W.ravel(), b]) for W, b in gate_layers(g)]).astype(np.float32)


# The paper's six-input gates (App. A.2).  "flux6": one MLP 6 -> 8 -> 8 -> 32 -> 1 over
# all six inputs; "wan6": a 3 -> 8 -> 8 branch on the budget inputs and one on the
# trajectory inputs, concatenated and fused by 16 -> 32 -> 1.  Layer shapes as (out, in).
GATE6_SHAPES = {
    "flux6": [(8, 6), (8, 8), (32, 8), (1, 32)],
    "wan6": [(8, 3), (8, 8), (8, 3), (8, 8), (32, 16), (1, 32)],
}


def gate_layers(g):
    """The (W, b) pairs of a six-input gate in evaluation / storage order."""
    return list(zip(g["W"], g["b"]))


def make_gate6(gate_seed, kind):
    """Seeded six-input gate: per layer W ~ U(-a, a) with a = sqrt(6 / (in + out)) and
    b ~ U(-0.1, 0.1); tensor keys 1, 2, ... in storage order (W1, b1, W2, b2, ...)."""
    Ws, bs = [], []
    key = 1
    for out, inn in GATE6_SHAPES[kind]:
        a = float(np.sqrt(6.0 / (inn + out)))
        Ws.append(uniform(gate_seed, key, out * inn, -a, a).reshape(out, inn))
        bs.append(uniform(gate_seed, key + 1, out, -0.1, 0.1))
        key += 2
    return {"kind": kind, "W": Ws, "b": bs, "mu": np.zeros(6, np.float32),
            "sd": np.ones(6, np.float32)}


def make_gate_any(gate_seed, kind="mlp3"):
    return make_gate(gate_seed) if kind == "mlp3" else make_gate6(gate_seed, kind)


# Sample inputs: latent noise, text tokens and pooled vector, all N(0, 1).
INPUT_KEYS = {"x": 1, "txt": 2, "pooled": 3, "txt_u": 4, "pooled_u": 5}


def make_inputs(cfg, sample_seed=0):
    seed = 1000 + cfg["weight_seed"] * 100 + sample_seed
    ni, nx, C, d = cfg["n_img"], cfg["n_txt"], cfg["patch_ch"], cfg["hidden"]
    x = normal(seed, INPUT_KEYS["x"], ni * C, 1.0).reshape(ni, C)
    txt = normal(seed, INPUT_KEYS["txt"], nx * d, 1.0).reshape(nx, d)
    pooled = normal(seed, INPUT_KEYS["pooled"], d, 1.0)
    # the unconditional branch of classifier-free guidance: its own text and pooled vector
    txt_u = normal(seed, INPUT_KEYS["txt_u"], nx * d, 1.0).reshape(nx, d)
    pooled_u = normal(seed, INPUT_KEYS["pooled_u"], d, 1.0)
    if cfg["dtype"] == "bf16":
        txt = bf16_round(txt)
        txt_u = bf16_round(txt_u)
    return {"x": x, "txt": txt, "pooled": pooled, "txt_u": txt_u, "pooled_u": pooled_u}
