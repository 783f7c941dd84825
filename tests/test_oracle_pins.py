"""Pins of the fp64 oracle against facts fixed by the paper and by mathematics.

Each test checks the oracle against something other than itself: closed forms,
invariants the paper states (Algorithm 2, Sec. 3.1-3.2), special cases that reduce to a
textbook routine, or brute force with scalar loops on tiny inputs.
"""

import itertools
import json
import math
import os

import numpy as np
import pytest

from oracle import bag_oracle as O
from paper_2608_09231_gb300 import configs, synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ---------------------------------------------------------------------------
# Algorithm 2: pacing
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("T", range(1, 11))
def test_pacing_spends_exactly_B_for_every_gate(T):
    """Algorithm 2 / Sec. 3.2: realized NFE = B exactly and m_0 = 1, whatever the gate."""
    for B in range(1, T + 1):
        for bits in itertools.product((0, 1), repeat=T - 1):
            m = O.schedule_from_gate_bits((None,) + bits, B, T)
            assert len(m) == T and m[0] == 1
            assert sum(m) == B
            # at a step where neither rule is forced, the gate's own bit stands
            c = 1
            for t in range(1, T):
                if c < B and B - c < T - t:
                    assert m[t] == bits[t - 1]
                c += m[t]


@pytest.mark.parametrize("T,B", [(10, 5), (50, 25), (50, 10), (7, 1), (7, 7), (12, 11)])
def test_pacing_closed_forms(T, B):
    """Adversarial gates have closed-form schedules: always-compute front-loads the
    budget, always-reuse leaves only the forced tail; B = T is all ones, B = 1 one-hot."""
    ones = O.schedule_from_gate_bits([None] + [1] * (T - 1), B, T)
    assert ones == [1] * B + [0] * (T - B)
    zeros = O.schedule_from_gate_bits([None] + [0] * (T - 1), B, T)
    assert zeros == [1] + [0] * (T - B) + [1] * (B - 1)
    if B == T:
        assert ones == zeros == [1] * T
    if B == 1:
        assert ones == zeros == [1] + [0] * (T - 1)


def test_alg2_rules_cannot_both_fire():
    """B - c = 0 and B - c >= T - t together would need T - t <= 0, impossible for t < T."""
    for T in range(1, 30):
        for t in range(1, T):
            for B in range(1, T + 1):
                for c in range(1, B + 1):
                    assert not (B - c >= T - t and B - c == 0)


def test_paper_speedups_are_nfe_ratios():
    """Tab. 3 quotes Qwen-Image speedups as NFE ratios: T / B at T = 50."""
    with open(os.path.join(GOLDEN, "paper_values.json")) as f:
        g = json.load(f)
    for row in g["qwen_nfe_speedups"]["rows"]:
        T, B, s = row["T"], row["B"], row["speedup"]
        m = O.schedule_from_gate_bits([None] + [0] * (T - 1), B, T)
        assert round(T / sum(m), 2) == s


# ---------------------------------------------------------------------------
# gate (Eq. 1) in float32
# ---------------------------------------------------------------------------
def _gate(seed=7):
    return synth.make_gate(seed)


def test_gate_param_count():
    g = _gate()
    n = synth.gate_flat(g).size
    assert n == 3 * 16 + 16 + 16 + 1 == 81  # under the paper's 1K-parameter bound (Sec. 3.2)


def test_gate_hand_example():
    """One active hidden unit: z = relu(f0) - 0.5 with f0 = (B - c)/B."""
    g = {"w1": np.zeros((16, 3), np.float32), "b1": np.zeros(16, np.float32),
         "w2": np.zeros(16, np.float32), "b2": np.array([-0.5], np.float32),
         "mu": np.zeros(3, np.float32), "sd": np.ones(3, np.float32)}
    g["w1"][0, 0] = 1.0
    g["w2"][0] = 1.0
    f = O.gate_features(B=4, T=10, c=1, t=3, drift=0.3)
    assert f[0] == np.float32(0.75) and f[1] == np.float32(0.7)
    assert O.gate_logit(f, g) == np.float32(0.25)
    f = O.gate_features(B=4, T=10, c=3, t=8, drift=0.3)
    assert O.gate_logit(f, g) == np.float32(-0.25)
    # the first input unit really is the first feature: moving it to input 2 reads drift
    g["w1"][0, 0], g["w1"][0, 2] = 0.0, 1.0
    assert O.gate_logit(f, g) == np.float32(0.3) - np.float32(0.5)


def test_gate_matches_fp64_matvec():
    """The fixed-order fp32 evaluation equals a float64 mat-vec up to fp32 rounding
    (pins the [out, in] indexing of W1 and the z-score direction)."""
    rng = np.random.default_rng(0)
    for seed in range(20):
        g = _gate(seed)
        g["mu"] = rng.normal(size=3).astype(np.float32) * 0.1
        g["sd"] = (1 + rng.random(3)).astype(np.float32)
        f = [np.float32(v) for v in rng.random(3)]
        z = O.gate_logit(f, g)
        fz = (np.array(f, np.float64) - g["mu"]) / g["sd"]
        h = np.maximum(g["w1"].astype(np.float64) @ fz + g["b1"], 0)
        z64 = float(g["w2"].astype(np.float64) @ h + g["b2"][0])
        assert abs(float(z) - z64) <= 1e-5 * (1 + abs(z64))


def test_gate_threshold_is_sigmoid_cutoff():
    """sigma(z) > tau  <=>  z > logit(tau) (Algorithm 2's cutoff), tau = 0.5 -> 0."""
    assert O.gate_threshold(0.5) == 0.0
    rng = np.random.default_rng(1)
    for tau in (0.3, 0.4, 0.5, 0.6, 0.7):
        thr = float(O.gate_threshold(tau))
        for z in rng.normal(size=200) * 3:
            if abs(z - thr) > 1e-5:
                assert (1 / (1 + math.exp(-z)) > tau) == (z > thr)


# ---------------------------------------------------------------------------
# elementwise pieces
# ---------------------------------------------------------------------------
def test_layer_norm_closed_form():
    x = np.array([[1.0, 2.0, 3.0, 4.0]])
    want = (x - 2.5) / math.sqrt(1.25 + 1e-6)
    assert np.allclose(O.layer_norm(x), want, rtol=0, atol=1e-15)
    y = O.layer_norm(np.random.default_rng(0).normal(size=(5, 64)) * 3 + 2)
    assert np.allclose(y.mean(-1), 0, atol=1e-12)
    assert np.allclose((y ** 2).mean(-1), 1, atol=1e-5)


def test_modulate_special_cases():
    rng = np.random.default_rng(0)
    xn, sh, sc = rng.normal(size=(3, 8)), rng.normal(size=8), rng.normal(size=8)
    assert np.array_equal(O.modulate(xn, 0.0, 0.0), xn)
    assert np.allclose(O.modulate(xn, sh, -np.ones(8)), np.broadcast_to(sh, (3, 8)))
    assert np.allclose(O.modulate(xn, sh, sc) - sh, xn * (1 + sc))


def test_gelu_tanh_against_erf_gelu():
    """The tanh form approximates x * Phi(x) to within 1e-3 everywhere."""
    xs = np.linspace(-8, 8, 4001)
    exact = np.array([0.5 * v * (1 + math.erf(v / math.sqrt(2))) for v in xs])
    assert np.max(np.abs(O.gelu_tanh(xs) - exact)) < 1e-3
    assert O.gelu_tanh(np.array([0.0]))[0] == 0.0
    assert abs(O.gelu_tanh(np.array([20.0]))[0] - 20.0) < 1e-12


def test_silu_closed_form():
    assert O.silu(np.array([0.0]))[0] == 0.0
    assert abs(O.silu(np.array([1.0]))[0] - 1 / (1 + math.exp(-1))) < 1e-15


def test_timestep_embedding():
    e0 = O.timestep_embedding(0.0)
    assert np.array_equal(e0, np.r_[np.ones(128), np.zeros(128)])
    t = 734.0
    e = O.timestep_embedding(t)
    assert abs(e[0] - math.cos(t)) < 1e-12 and abs(e[128] - math.sin(t)) < 1e-12
    # frequencies form a geometric sequence from 1 down to 10000^(-127/128)
    fr = np.arctan2(O.timestep_embedding(1e-3)[128:], O.timestep_embedding(1e-3)[:128]) / 1e-3
    assert np.allclose(fr[1:] / fr[:-1], 10000 ** (-1 / 128), rtol=1e-6)
    assert np.allclose(e[:128] ** 2 + e[128:] ** 2, 1)


def test_sigma_grid():
    s = O.sigma_grid(50)
    assert s[0] == 1.0 and s[-1] == 0.0 and np.allclose(np.diff(s), -1 / 50)


def test_linear_against_loops():
    rng = np.random.default_rng(0)
    x, w, b = rng.normal(size=(3, 5)), rng.normal(size=(4, 5)), rng.normal(size=4)
    y = O.linear(x, w, b)
    for i in range(3):
        for o in range(4):
            assert abs(y[i, o] - (b[o] + sum(x[i, k] * w[o, k] for k in range(5)))) < 1e-12


def test_rel_l1():
    a, b = np.array([1.0, 2.0]), np.array([2.0, 2.0])
    assert O.rel_l1(a, b) == 0.25
    rng = np.random.default_rng(0)
    x, y = rng.normal(size=100), rng.normal(size=100)
    assert O.rel_l1(x, x) == 0.0
    assert abs(O.rel_l1(3.5 * x, 3.5 * y) - O.rel_l1(x, y)) < 1e-12


# ---------------------------------------------------------------------------
# RoPE and attention
# ---------------------------------------------------------------------------
def test_rope_identity_at_origin_and_norm_preserving():
    rng = np.random.default_rng(0)
    x = rng.normal(size=(6, 2, 128))
    pos = np.zeros((6, 3))
    assert np.array_equal(O.apply_rope(x, O.rope_angles(pos, (16, 56, 56))), x)
    pos = rng.integers(0, 80, size=(6, 3)).astype(float)
    y = O.apply_rope(x, O.rope_angles(pos, (16, 56, 56)))
    assert np.allclose(np.linalg.norm(y, axis=-1), np.linalg.norm(x, axis=-1))


def test_rope_first_pair_turns_by_position():
    """Pair 0 of each axis has frequency 1: e_0 at position p becomes (cos p, sin p)."""
    x = np.zeros((1, 1, 64))
    x[0, 0, 0] = 1.0
    y = O.apply_rope(x, O.rope_angles(np.array([[0.0, 3.0, 5.0]]), (0, 32, 32)))
    assert abs(y[0, 0, 0] - math.cos(3)) < 1e-15 and abs(y[0, 0, 1] - math.sin(3)) < 1e-15
    x = np.zeros((1, 1, 64))
    x[0, 0, 32] = 1.0  # first pair of the column axis
    y = O.apply_rope(x, O.rope_angles(np.array([[0.0, 3.0, 5.0]]), (0, 32, 32)))
    assert abs(y[0, 0, 32] - math.cos(5)) < 1e-15 and abs(y[0, 0, 33] - math.sin(5)) < 1e-15


def test_rope_scores_depend_on_relative_position_only():
    rng = np.random.default_rng(1)
    q, k = rng.normal(size=(1, 1, 128)), rng.normal(size=(1, 1, 128))
    axes = (16, 56, 56)
    p, p2 = np.array([[1.0, 7.0, 3.0]]), np.array([[0.0, 2.0, 9.0]])
    s = np.array([[4.0, -5.0, 11.0]])
    a = np.sum(O.apply_rope(q, O.rope_angles(p, axes)) * O.apply_rope(k, O.rope_angles(p2, axes)))
    b = np.sum(O.apply_rope(q, O.rope_angles(p + s, axes)) *
               O.apply_rope(k, O.rope_angles(p2 + s, axes)))
    assert abs(a - b) < 1e-9


def _attention_loops(q, k, v):
    N, H, D = q.shape
    M = k.shape[0]
    out = np.zeros((N, H, D))
    for h in range(H):
        for i in range(N):
            s = [sum(q[i, h, e] * k[j, h, e] for e in range(D)) / math.sqrt(D) for j in range(M)]
            mx = max(s)
            w = [math.exp(x - mx) for x in s]
            tot = sum(w)
            for e in range(D):
                out[i, h, e] = sum(w[j] * v[j, h, e] for j in range(M)) / tot
    return out


def test_attention_brute_force_and_rows_sum_to_one():
    rng = np.random.default_rng(0)
    q, k, v = rng.normal(size=(5, 2, 4)), rng.normal(size=(7, 2, 4)), rng.normal(size=(7, 2, 4))
    assert np.allclose(O.attention(q, k, v), _attention_loops(q, k, v), atol=1e-12)
    p = O.softmax_rows(rng.normal(size=(9, 13)) * 10)
    assert np.allclose(p.sum(-1), 1) and (p >= 0).all()
    # equal keys -> uniform weights -> mean of v
    kk = np.repeat(rng.normal(size=(1, 2, 4)), 7, axis=0)
    assert np.allclose(O.attention(q, kk, v), np.broadcast_to(v.mean(0), (5, 2, 4)))
    # a large-valued row stays finite (max subtraction)
    assert np.isfinite(O.softmax_rows(np.array([[1e4, 0.0, -1e4]]))).all()


# ---------------------------------------------------------------------------
# blocks: brute force with scalar loops on tiny shapes
# ---------------------------------------------------------------------------
def _ln_loop(row, eps=1e-6):
    n = len(row)
    mu = sum(row) / n
    var = sum((x - mu) ** 2 for x in row) / n
    return [(x - mu) / math.sqrt(var + eps) for x in row]


def _lin_loop(rows, w, b):
    return [[b[o] + sum(r[i] * w[o][i] for i in range(len(r))) for o in range(len(w))]
            for r in rows]


def _gelu(x):
    return 0.5 * x * (1 + math.tanh(math.sqrt(2 / math.pi) * (x + 0.044715 * x ** 3)))


def _rope_loop(vec, angs):
    out = list(vec)
    for j, a in enumerate(angs):
        x0, x1 = vec[2 * j], vec[2 * j + 1]
        out[2 * j] = x0 * math.cos(a) - x1 * math.sin(a)
        out[2 * j + 1] = x0 * math.sin(a) + x1 * math.cos(a)
    return out


def _attn_rows(q, k, v, H):
    """q, k, v as lists of rows [N][d]; heads are contiguous column slices."""
    d = len(q[0])
    D = d // H
    out = [[0.0] * d for _ in q]
    for h in range(H):
        sl = range(h * D, (h + 1) * D)
        for i in range(len(q)):
            s = [sum(q[i][e] * k[j][e] for e in sl) / math.sqrt(D) for j in range(len(k))]
            mx = max(s)
            w = [math.exp(x - mx) for x in s]
            tot = sum(w)
            for e in sl:
                out[i][e] = sum(w[j] * v[j][e] for j in range(len(k))) / tot
    return out


def _rand_block(rng, shapes):
    return {n: rng.normal(size=s) * (0.3 if len(s) == 2 else 0.2) for n, s in shapes.items()}


def _head_angles(ang, H):
    return [list(a) * 1 for a in ang]


def _rms_loop(vec, w, eps=1e-6):
    ms = sum(x * x for x in vec) / len(vec)
    return [x / math.sqrt(ms + eps) * w[i] for i, x in enumerate(vec)]


def _qk_loop(r, off, D, H, W, name, ang_i):
    """Heads of one projected row at column offset off: RMS-normalised with W[name]
    (when present) and then rotated."""
    out = []
    for hh in range(H):
        x = r[off + hh * D:off + (hh + 1) * D]
        if name in W:
            x = _rms_loop(x, W[name].tolist())
        out += _rope_loop(x, ang_i)
    return out


@pytest.mark.parametrize("qkn", [False, True])
def test_single_block_brute_force(qkn):
    rng = np.random.default_rng(3)
    N, d, H, F = 5, 8, 2, 12
    cfg = {"hidden": d, "mlp": F, "heads": H, "qk_norm": qkn}
    W = _rand_block(rng, synth.block_shapes(cfg, "single"))
    h = rng.normal(size=(N, d))
    mod = rng.normal(size=3 * d) * 0.5
    pos = rng.integers(0, 5, size=(N, 3)).astype(float)
    ang = O.rope_angles(pos, (0, 2, 2))
    got = O.single_block(h, mod, W, ang, H)
    sh, sc, g = mod[:d], mod[d:2 * d], mod[2 * d:]
    xn = [[v * (1 + sc[i]) + sh[i] for i, v in enumerate(_ln_loop(list(r)))] for r in h]
    y = _lin_loop(xn, W["lin1_w"].tolist(), W["lin1_b"].tolist())
    D = d // H
    q = [_qk_loop(r, 0, D, H, W, "q_norm", ang[i]) for i, r in enumerate(y)]
    k = [_qk_loop(r, d, D, H, W, "k_norm", ang[i]) for i, r in enumerate(y)]
    v = [r[2 * d:3 * d] for r in y]
    a = _attn_rows(q, k, v, H)
    cat = [a[i] + [_gelu(x) for x in y[i][3 * d:]] for i in range(N)]
    o = _lin_loop(cat, W["lin2_w"].tolist(), W["lin2_b"].tolist())
    want = np.array([[h[i, j] + g[j] * o[i][j] for j in range(d)] for i in range(N)])
    assert np.allclose(got, want, atol=1e-12)
    # sampled-row evaluation agrees with the full evaluation
    assert np.allclose(O.single_block(h, mod, W, ang, H, rows=[4, 1]), got[[4, 1]], atol=1e-13)


@pytest.mark.parametrize("qkn", [False, True])
def test_double_block_brute_force(qkn):
    rng = np.random.default_rng(4)
    ni, nx, d, H, F = 4, 3, 8, 2, 12
    W = _rand_block(rng, synth.block_shapes({"hidden": d, "mlp": F, "heads": H, "qk_norm": qkn},
                                            "double"))
    img, txt = rng.normal(size=(ni, d)), rng.normal(size=(nx, d))
    mi, mt = rng.normal(size=6 * d) * 0.5, rng.normal(size=6 * d) * 0.5
    pos = np.concatenate([np.zeros((nx, 3)), rng.integers(0, 4, size=(ni, 3))]).astype(float)
    ang = O.rope_angles(pos, (0, 2, 2))
    gi, gt = O.double_block(img, txt, mi, mt, W, ang, H)

    def mods(m):
        return [m[i * d:(i + 1) * d] for i in range(6)]

    Mi, Mt = mods(mi), mods(mt)

    def lnmod(rows, sh, sc):
        return [[v * (1 + sc[i]) + sh[i] for i, v in enumerate(_ln_loop(list(r)))] for r in rows]

    qkv_t = _lin_loop(lnmod(txt, Mt[0], Mt[1]), W["txt_qkv_w"].tolist(), W["txt_qkv_b"].tolist())
    qkv_i = _lin_loop(lnmod(img, Mi[0], Mi[1]), W["img_qkv_w"].tolist(), W["img_qkv_b"].tolist())
    joint = qkv_t + qkv_i
    D = d // H
    pre = ["txt_"] * nx + ["img_"] * ni
    q = [_qk_loop(r, 0, D, H, W, pre[i] + "q_norm", ang[i]) for i, r in enumerate(joint)]
    k = [_qk_loop(r, d, D, H, W, pre[i] + "k_norm", ang[i]) for i, r in enumerate(joint)]
    v = [r[2 * d:] for r in joint]
    a = _attn_rows(q, k, v, H)

    def stream(x, a_s, M, pre):
        o = _lin_loop(a_s, W[pre + "_proj_w"].tolist(), W[pre + "_proj_b"].tolist())
        x = [[x[i][j] + M[2][j] * o[i][j] for j in range(d)] for i in range(len(x))]
        u = _lin_loop(lnmod(x, M[3], M[4]), W[pre + "_up_w"].tolist(), W[pre + "_up_b"].tolist())
        dn = _lin_loop([[_gelu(t) for t in r] for r in u], W[pre + "_down_w"].tolist(),
                       W[pre + "_down_b"].tolist())
        return np.array([[x[i][j] + M[5][j] * dn[i][j] for j in range(d)] for i in range(len(x))])

    assert np.allclose(gt, stream(txt.tolist(), a[:nx], Mt, "txt"), atol=1e-12)
    assert np.allclose(gi, stream(img.tolist(), a[nx:], Mi, "img"), atol=1e-12)


def test_wan_block_brute_force():
    rng = np.random.default_rng(5)
    ni, nx, d, H, F = 5, 3, 8, 2, 10
    W = _rand_block(rng, synth.block_shapes({"hidden": d, "mlp": F}, "wan"))
    x, ctx = rng.normal(size=(ni, d)), rng.normal(size=(nx, d))
    e = rng.normal(size=6 * d) * 0.5
    ang = O.rope_angles(rng.integers(0, 4, size=(ni, 3)).astype(float), (2, 0, 2))
    got = O.wan_block(x, ctx, e, W, ang, H)
    M = [e[i * d:(i + 1) * d] for i in range(6)]
    D = d // H

    def lnmod(rows, sh, sc):
        return [[v * (1 + sc[i]) + sh[i] for i, v in enumerate(_ln_loop(list(r)))] for r in rows]

    y = _lin_loop(lnmod(x, M[0], M[1]), W["sa_qkv_w"].tolist(), W["sa_qkv_b"].tolist())
    q = [sum((_rope_loop(r[hh * D:(hh + 1) * D], ang[i]) for hh in range(H)), [])
         for i, r in enumerate(y)]
    k = [sum((_rope_loop(r[d + hh * D:d + (hh + 1) * D], ang[i]) for hh in range(H)), [])
         for i, r in enumerate(y)]
    v = [r[2 * d:] for r in y]
    o = _lin_loop(_attn_rows(q, k, v, H), W["sa_o_w"].tolist(), W["sa_o_b"].tolist())
    xs = [[x[i, j] + M[2][j] * o[i][j] for j in range(d)] for i in range(ni)]
    qc = _lin_loop([_ln_loop(r) for r in xs], W["ca_q_w"].tolist(), W["ca_q_b"].tolist())
    kv = _lin_loop(ctx.tolist(), W["ca_kv_w"].tolist(), W["ca_kv_b"].tolist())
    oc = _lin_loop(_attn_rows(qc, [r[:d] for r in kv], [r[d:] for r in kv], H),
                   W["ca_o_w"].tolist(), W["ca_o_b"].tolist())
    xs = [[xs[i][j] + oc[i][j] for j in range(d)] for i in range(ni)]
    u = _lin_loop(lnmod(xs, M[3], M[4]), W["ffn_up_w"].tolist(), W["ffn_up_b"].tolist())
    dn = _lin_loop([[_gelu(t) for t in r] for r in u], W["ffn_down_w"].tolist(),
                   W["ffn_down_b"].tolist())
    want = np.array([[xs[i][j] + M[5][j] * dn[i][j] for j in range(d)] for i in range(ni)])
    assert np.allclose(got, want, atol=1e-12)


def test_row_restricted_blocks_equal_full_evaluation():
    """Evaluating a block at a subset of rows gives those rows of the full evaluation."""
    rng = np.random.default_rng(8)
    d, H, F, ni, nx = 8, 2, 12, 5, 3
    Wd = _rand_block(rng, synth.block_shapes({"hidden": d, "mlp": F}, "double"))
    img, txt = rng.normal(size=(ni, d)), rng.normal(size=(nx, d))
    mi, mt = rng.normal(size=6 * d) * 0.5, rng.normal(size=6 * d) * 0.5
    ang = O.rope_angles(np.concatenate([np.zeros((nx, 3)), rng.integers(0, 4, size=(ni, 3))]),
                        (0, 2, 2))
    gi, gt = O.double_block(img, txt, mi, mt, Wd, ang, H)
    full = np.concatenate([gt, gi])
    rows = [6, 0, 2, 4]
    assert np.allclose(O.double_block(img, txt, mi, mt, Wd, ang, H, rows=rows), full[rows],
                       atol=1e-13)
    Ww = _rand_block(rng, synth.block_shapes({"hidden": d, "mlp": F}, "wan"))
    e = rng.normal(size=6 * d) * 0.5
    angw = O.rope_angles(rng.integers(0, 4, size=(ni, 3)).astype(float), (2, 0, 2))
    fw = O.wan_block(img, txt, e, Ww, angw, H)
    assert np.allclose(O.wan_block(img, txt, e, Ww, angw, H, rows=[3, 1]), fw[[3, 1]], atol=1e-13)


def test_zero_gate_blocks_are_identity():
    rng = np.random.default_rng(6)
    d, H, F = 8, 2, 12
    W = _rand_block(rng, synth.block_shapes({"hidden": d, "mlp": F}, "single"))
    h = rng.normal(size=(4, d))
    mod = np.r_[rng.normal(size=2 * d), np.zeros(d)]
    ang = O.rope_angles(np.zeros((4, 3)), (0, 2, 2))
    assert np.array_equal(O.single_block(h, mod, W, ang, H), h)


# ---------------------------------------------------------------------------
# the sampler: Algorithm 2 end to end on the tiny stack
# ---------------------------------------------------------------------------
def _tiny(**kw):
    cfg = configs.get_config("tiny", **kw)
    return cfg, synth.make_weights(cfg), synth.make_gate(cfg["gate_seed"]), synth.make_inputs(cfg)


def test_budget_equal_T_reproduces_uncached_sampling_exactly():
    """Sec. 3.1: the all-ones schedule is the full-compute target x_T(1, p)."""
    cfg, W, g, inp = _tiny(grid=(1, 6, 6), n_txt=5)
    T = 6
    a = O.sample(cfg, W, g, inp, T=T, B=T)
    b = O.sample(cfg, W, g, inp, T=T, B=1, policy="full")
    assert a["mask"] == [1] * T and a["nfe"] == T
    assert np.array_equal(a["x"], b["x"])


@pytest.mark.parametrize("tau", [0.3, 0.5, 0.7])
def test_nfe_equals_budget_for_any_tau(tau):
    """App. C tau sweep: the cutoff moves placements, never the cost."""
    cfg, W, g, inp = _tiny(grid=(1, 5, 5), n_txt=4)
    for B in (1, 3, 6):
        r = O.sample(cfg, W, g, inp, T=6, B=B, tau=tau)
        assert r["nfe"] == B and sum(r["mask"]) == B and r["mask"][0] == 1


def test_same_gate_runs_at_other_step_counts():
    """Sec. 4.3: the gate's inputs are ratios, so one checkpoint runs at T = 25, 28, 50."""
    cfg, W, g, inp = _tiny(grid=(1, 3, 3), n_txt=2, hidden=64, heads=1, mlp=64,
                           rope_axes=(0, 32, 32))
    for T, B in ((25, 9), (28, 13), (50, 20)):
        r = O.sample(cfg, W, g, inp, T=T, B=B)
        assert r["nfe"] == B and len(r["mask"]) == T


def _constant_offset_net(cfg, W):
    """Make every block add a step-independent vector to the stream: time MLP input
    weights zero (conditioning constant in t), lin2 weights zero (block output = bias)."""
    W["global"]["t1_w"][:] = 0.0
    for blk in W["blocks"]:
        blk["lin2_w"][:] = 0.0
    return W


def test_reused_step_is_input_plus_cached_residual():
    """Residual reuse (Sec. 2, Algorithm 2): when the stack adds a constant vector, the
    cached residual equals what a full step would add, so any schedule reproduces the
    uncached latent."""
    cfg, W, g, inp = _tiny(grid=(1, 5, 5), n_txt=4)
    W = _constant_offset_net(cfg, W)
    full = O.sample(cfg, W, g, inp, T=7, B=7)["x"]
    for mask in ([1, 0, 0, 0, 0, 0, 0], [1, 0, 1, 0, 0, 1, 0], [1, 1, 0, 1, 0, 1, 1]):
        r = O.sample(cfg, W, g, inp, T=7, B=sum(mask), policy=mask)
        assert r["mask"] == mask
        assert np.allclose(r["x"], full, atol=1e-12)
    # ... and an input-dependent stack does notice the reuse
    cfg, W, g, inp = _tiny(grid=(1, 5, 5), n_txt=4)
    a = O.sample(cfg, W, g, inp, T=7, B=7)["x"]
    b = O.sample(cfg, W, g, inp, T=7, B=2, policy=[1, 0, 0, 0, 0, 0, 1])["x"]
    assert not np.allclose(a, b, atol=1e-6)


def test_euler_closed_form_for_constant_velocity():
    """sum over steps of (sigma_{t+1} - sigma_t) = -1, so a constant velocity b gives
    x_T = x_0 - b."""
    cfg, W, g, inp = _tiny(grid=(1, 4, 4), n_txt=3)
    W["global"]["fin_w"][:] = 0.0
    r = O.sample(cfg, W, g, inp, T=9, B=4)
    assert np.allclose(r["x"], inp["x"] - W["global"]["fin_b"][None, :], atol=1e-12)


def test_conditioning_closed_form():
    cfg, W, g, inp = _tiny()
    G = O.to64(W)["global"]
    G["t1_w"][:] = 0.0
    G["t2_w"][:] = 0.0
    vec = O.conditioning(cfg, G, 0.3, inp["pooled"].astype(np.float64))
    assert np.allclose(vec, G["t2_b"] + inp["pooled"])


def _conditioning_loops(sigma, t1_w, t1_b, t2_w, t2_b, pooled):
    """Scalar-loop conditioning vector: the 256-wide sinusoid of 1000 sigma (cos half,
    then sin half, frequencies 10000^(-j/128)), a dense layer t1, SiLU, a dense layer t2
    (weights stored [out][in]), plus the pooled text vector when one is given."""
    tval = 1000.0 * sigma
    e = [math.cos(tval * math.exp(-math.log(10000.0) * j / 128)) for j in range(128)]
    e += [math.sin(tval * math.exp(-math.log(10000.0) * j / 128)) for j in range(128)]
    h = []
    for o in range(len(t1_b)):
        acc = t1_b[o]
        for i in range(256):
            acc += t1_w[o][i] * e[i]
        h.append(acc / (1.0 + math.exp(-acc)))
    out = []
    for o in range(len(t2_b)):
        acc = t2_b[o]
        for i in range(len(h)):
            acc += t2_w[o][i] * h[i]
        out.append(acc + (pooled[o] if pooled is not None else 0.0))
    return out


@pytest.mark.parametrize("kind", ["single", "wan"])
def test_conditioning_brute_force(kind):
    """The whole conditioning chain with non-zero weights against scalar loops; for the
    Wan kind the pooled vector must not enter (time embedding only)."""
    d = 8
    rng = np.random.default_rng(7)
    G = {"t1_w": rng.normal(0, 0.3, (d, 256)), "t1_b": rng.normal(0, 0.3, d),
         "t2_w": rng.normal(0, 0.5, (d, d)), "t2_b": rng.normal(0, 0.3, d)}
    pooled = rng.normal(0, 1, d)
    cfg = {"kind": kind}
    for sigma in (1.0, 0.37, 0.02):
        got = O.conditioning(cfg, G, sigma, pooled)
        want = _conditioning_loops(sigma, G["t1_w"].tolist(), G["t1_b"].tolist(),
                                   G["t2_w"].tolist(), G["t2_b"].tolist(),
                                   None if kind == "wan" else pooled.tolist())
        assert np.allclose(got, want, rtol=1e-12, atol=1e-12), (kind, sigma)


def test_conditioning_detects_plausible_mistakes():
    """Dropping the SiLU, swapping the two layers' roles or transposing t1 each change the
    vector by far more than rounding (the brute force above would catch them)."""
    d = 8
    rng = np.random.default_rng(11)
    G = {"t1_w": rng.normal(0, 0.3, (d, 256)), "t1_b": rng.normal(0, 0.3, d),
         "t2_w": rng.normal(0, 0.5, (d, d)), "t2_b": rng.normal(0, 0.3, d)}
    pooled = rng.normal(0, 1, d)
    cfg = {"kind": "single"}
    got = np.array(O.conditioning(cfg, G, 0.6, pooled))
    e = O.timestep_embedding(600.0)
    no_silu = G["t2_w"] @ (G["t1_w"] @ e + G["t1_b"]) + G["t2_b"] + pooled
    silu_after = O.silu(G["t2_w"] @ (G["t1_w"] @ e + G["t1_b"]) + G["t2_b"]) + pooled
    no_pooled = got - pooled
    for wrong in (no_silu, silu_after, no_pooled):
        assert np.max(np.abs(got - wrong)) > 1e-3


def test_embedded_observable_closed_form_on_constant_velocity_net():
    """The paper's observable (Eq. 3): the post-patch-embedding tokens.  With the final
    layer's weight zeroed the velocity is the constant bias b at every step, so
    x_t = x_0 + (sigma_t - 1) b and every row of h_t - h_s equals
    (sigma_t - sigma_s) W_pe b: the drift and the step change have closed forms."""
    cfg, W, g, inp = _tiny(grid=(1, 6, 6), n_txt=5, observable="embedded")
    W["global"]["fin_w"][:] = 0.0
    T, B = 8, 4
    r = O.sample(cfg, W, g, inp, T=T, B=B)
    G = O.to64(W)["global"]
    sig = O.sigma_grid(T)
    b = G["fin_b"]
    x0 = inp["x"].astype(np.float64)
    u = G["pe_w"] @ b
    n = x0.shape[0]

    def h(t):
        return (x0 + (sig[t] - 1.0) * b) @ G["pe_w"].T + G["pe_b"]

    last = 0
    for t in range(1, T):
        drift = n * abs(sig[t] - sig[last]) * np.abs(u).sum() / np.abs(h(last)).sum()
        step = n * abs(sig[t] - sig[t - 1]) * np.abs(u).sum() / np.abs(h(t - 1)).sum()
        rec = r["log"][t]
        assert abs(rec["drift"] - drift) <= 1e-12 * max(1.0, drift), t
        assert abs(rec["s_traj"][2] - step) <= 1e-12 * max(1.0, step), t
        assert rec["s_traj"][0] == t - last
        if r["mask"][t]:
            last = t
    # the default observable (block 0's modulated input) reads something else
    r2 = O.sample(dict(cfg, observable="modulated"), W, g, inp, T=T, B=B, policy=r["mask"])
    assert abs(r2["log"][1]["drift"] - r["log"][1]["drift"]) > 1e-6


def test_observable_selects_the_embedded_tokens_or_the_modulated_input():
    """At one step the embedded observable is the patch-embedded tensor itself, whatever
    the blocks hold; the default is the first block's LayerNorm-modulated image stream."""
    cfg, W, g, inp = _tiny(grid=(1, 6, 6), n_txt=5)
    W64 = O.to64(W)
    G, blocks = W64["global"], W64["blocks"]
    vec = O.conditioning(cfg, G, 0.7, inp["pooled"].astype(np.float64))
    h = O.patch_embed(G, inp["x"].astype(np.float64))
    emb = O.observable(dict(cfg, observable="embedded"), G, blocks, vec, h)
    assert emb is h
    mod = O.observable(cfg, G, blocks, vec, h)
    assert np.array_equal(mod, O.first_modulated_input(cfg, G, blocks, vec, h))
    assert np.max(np.abs(mod - h)) > 0.1


def test_drift_is_zero_when_nothing_moves_and_logged_features():
    """With the velocity forced to zero the latent never moves, so the first block's
    modulated input changes only through the time embedding; with that frozen too the
    drift is exactly zero at every step."""
    cfg, W, g, inp = _tiny(grid=(1, 4, 4), n_txt=3)
    W["global"]["fin_w"][:] = 0.0
    W["global"]["fin_b"][:] = 0.0
    W["global"]["t1_w"][:] = 0.0
    r = O.sample(cfg, W, g, inp, T=5, B=3)
    for rec in r["log"][1:]:
        assert rec["drift"] == 0.0
        assert rec["s_traj"][0] == rec["t"] - max(
            q["t"] for q in r["log"][:rec["t"]] if q["full"])
        assert rec["features"][0] == np.float32(3 - rec["c_before"]) / np.float32(3)


# ---------------------------------------------------------------------------
# the paper's six-input gates (App. A.2) and the full state of Eq. 3
# ---------------------------------------------------------------------------
def test_six_input_gate_parameter_counts_match_the_paper():
    with open(os.path.join(GOLDEN, "paper_values.json")) as f:
        want = json.load(f)["gate_param_counts"]
    assert synth.gate_flat(synth.make_gate6(5, "flux6")).size == want["flux"] == 449
    assert synth.gate_flat(synth.make_gate6(5, "wan6")).size == want["wan"] == 785


def test_six_features_closed_form():
    f = O.gate_features6(B=20, T=50, c=5, t=10, t_last=7, drift=0.125, step=0.0625)
    assert f == [np.float32(0.4), np.float32(0.75), np.float32(15) / np.float32(40),
                 np.float32(3.0), np.float32(0.125), np.float32(0.0625)]


def _relu(x):
    return np.maximum(x, 0.0)


@pytest.mark.parametrize("kind", ["flux6", "wan6"])
def test_six_input_gate_matches_fp64_forward(kind):
    """Fixed-order fp32 evaluation equals a float64 forward pass to rounding; the fp64
    pass spells out the architecture (layer order; Wan: budget branch on inputs 0-2,
    trajectory branch on 3-5, concatenated budget-first)."""
    rng = np.random.default_rng(2)
    for seed in range(10):
        g = synth.make_gate6(seed, kind)
        g["mu"] = (rng.normal(size=6) * 0.1).astype(np.float32)
        g["sd"] = (1 + rng.random(6)).astype(np.float32)
        f = [np.float32(v) for v in rng.random(6) * 2]
        z = float(O.gate_logit6(f, g))
        x = (np.array(f, np.float64) - g["mu"]) / g["sd"]
        Ws = [w.astype(np.float64) for w in g["W"]]
        bs = [b.astype(np.float64) for b in g["b"]]
        if kind == "flux6":
            h = x
            for k in range(3):
                h = _relu(Ws[k] @ h + bs[k])
            z64 = float((Ws[3] @ h + bs[3])[0])
        else:
            hb = _relu(Ws[1] @ _relu(Ws[0] @ x[:3] + bs[0]) + bs[1])
            ht = _relu(Ws[3] @ _relu(Ws[2] @ x[3:] + bs[2]) + bs[3])
            z64 = float((Ws[5] @ _relu(Ws[4] @ np.r_[hb, ht] + bs[4]) + bs[5])[0])
        assert abs(z - z64) <= 1e-5 * (1 + abs(z64))


def test_wan_gate_branches_read_their_own_inputs():
    """With only the trajectory branch's path to the output open and identity-like
    weights, z = relu(t - t_last) - 2: the branch reads input 3 (staleness)."""
    g = synth.make_gate6(1, "wan6")
    for W in g["W"]:
        W[:] = 0.0
    for b in g["b"]:
        b[:] = 0.0
    g["W"][2][0, 0] = 1.0      # trajectory branch layer 1: input 0 of its slice = t - t_last
    g["W"][3][0, 0] = 1.0      # trajectory branch layer 2
    g["W"][4][0, 8] = 1.0      # fuse layer reads the first trajectory feature (index 8)
    g["W"][5][0, 0] = 1.0
    g["b"][5][0] = -2.0
    f = O.gate_features6(B=20, T=50, c=5, t=10, t_last=7, drift=0.5, step=0.5)
    assert O.gate_logit6(f, g) == np.float32(1.0)
    f = O.gate_features6(B=20, T=50, c=5, t=10, t_last=9, drift=0.5, step=0.5)
    assert O.gate_logit6(f, g) == np.float32(-1.0)


@pytest.mark.parametrize("kind", ["flux6", "wan6"])
def test_six_input_gates_spend_exactly_B(kind):
    cfg, W, _, inp = _tiny(grid=(1, 4, 4), n_txt=3)
    g = synth.make_gate6(cfg["gate_seed"], kind)
    for B in (1, 4, 7):
        r = O.sample(cfg, W, g, inp, T=7, B=B)
        assert r["nfe"] == B and r["mask"][0] == 1
        for rec in r["log"][1:]:
            assert len(rec["features"]) == 6
            assert rec["features"][3] == rec["s_traj"][0]


# ---------------------------------------------------------------------------
# the two other scheduling paradigms of Sec. 3.1 on the same signal path
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("T", [1, 7, 10, 50])
def test_static_uniform_schedule_closed_form(T):
    for B in range(1, T + 1):
        m = O.static_uniform_schedule(B, T)
        assert sum(m) == B and m[0] == 1
        on = [t for t in range(T) if m[t]]
        gaps = {b - a for a, b in zip(on, on[1:])}
        assert gaps <= {T // B, -(-T // B)}       # spacing floor(T/B) or ceil(T/B)
    assert O.static_uniform_schedule(5, 50) == [1 if t % 10 == 0 else 0 for t in range(50)]


def test_threshold_policy_extremes():
    """q_t >= 0, so delta < 0 computes every step and a huge delta only step 0; the
    realised NFE is whatever the rule gives (no budget enters)."""
    cfg, W, g, inp = _tiny(grid=(1, 4, 4), n_txt=3)
    r = O.sample(cfg, W, g, inp, T=6, B=2, policy=("threshold", -1.0))
    assert r["mask"] == [1] * 6 and r["nfe"] == 6
    r = O.sample(cfg, W, g, inp, T=6, B=2, policy=("threshold", 1e9))
    assert r["mask"] == [1, 0, 0, 0, 0, 0] and r["nfe"] == 1
    r = O.sample(cfg, W, g, inp, T=6, B=2, policy="uniform")
    assert r["mask"] == [1, 0, 0, 1, 0, 0]


# ---------------------------------------------------------------------------
# classifier-free guidance with one shared mask (App. A.1)
# ---------------------------------------------------------------------------
def test_guidance_special_cases():
    """g = 1 gives v = v_c (the conditional sampler); identical branches give v = v_c
    for any g, bit for bit; the shared mask spends exactly B and depends only on the
    conditional branch's signal."""
    cfg, W, g, inp = _tiny(grid=(1, 4, 4), n_txt=3)
    T, B = 6, 3
    base = O.sample(cfg, W, g, inp, T=T, B=B)
    one = O.sample(cfg, W, g, inp, T=T, B=B, guidance=1.0)
    assert one["mask"] == base["mask"]
    assert np.allclose(one["x"], base["x"], atol=1e-12)
    same = dict(inp, txt_u=inp["txt"], pooled_u=inp["pooled"])
    r = O.sample(cfg, W, g, same, T=T, B=B, guidance=4.5)
    assert np.array_equal(r["x"], base["x"]) and r["mask"] == base["mask"]
    r = O.sample(cfg, W, g, inp, T=T, B=B, guidance=4.5)
    assert r["nfe"] == B and r["mask"] == base["mask"]   # decisions read the cond branch
    assert not np.allclose(r["x"], base["x"], atol=1e-6)


def test_guidance_reuse_is_per_branch_residual():
    """With a stack that adds a step-independent vector per branch, any shared schedule
    reproduces the uncached guided latent: each branch reuses its own residual."""
    cfg, W, g, inp = _tiny(grid=(1, 4, 4), n_txt=3)
    W = _constant_offset_net(cfg, W)
    full = O.sample(cfg, W, g, inp, T=6, B=6, guidance=3.0)["x"]
    r = O.sample(cfg, W, g, inp, T=6, B=3, guidance=3.0, policy=[1, 0, 0, 1, 0, 1])
    assert np.allclose(r["x"], full, atol=1e-12)


# ---------------------------------------------------------------------------
# QK-RMSNorm (FLUX / Qwen-Image blocks)
# ---------------------------------------------------------------------------
def test_rms_norm_heads_closed_forms():
    """Unit scale: every head comes out with RMS 1 (up to eps); the result does not
    depend on the input's scale; for zero-mean heads it equals LayerNorm; the scale
    multiplies channel by channel."""
    rng = np.random.default_rng(11)
    x = rng.normal(size=(6, 3, 16)) * 5
    y = O.rms_norm_heads(x, np.ones(16), eps=0.0)
    assert np.allclose(np.sqrt(np.mean(y ** 2, axis=-1)), 1.0, atol=1e-14)
    assert np.allclose(O.rms_norm_heads(7.5 * x, np.ones(16), eps=0.0), y, atol=1e-13)
    z = x - x.mean(axis=-1, keepdims=True)
    assert np.allclose(O.rms_norm_heads(z, np.ones(16)),
                       O.layer_norm(z.reshape(-1, 16)).reshape(z.shape), atol=1e-12)
    w = rng.normal(size=16)
    assert np.allclose(O.rms_norm_heads(x, w, eps=0.0), y * w, atol=1e-13)


def test_qk_norm_weights_and_block_use():
    """The generator's norm scales are 1 + N(0, 0.02) per head channel; a block with unit
    scales attends with unit-RMS q and k heads; removing the scales gives the plain block."""
    cfg = configs.get_config("flux_small", qk_norm=True)
    W = synth.make_weights(cfg, blocks=[0, cfg["n_double"]])
    b = W["blocks"][0]
    for n in ("img_q_norm", "img_k_norm", "txt_q_norm", "txt_k_norm"):
        assert b[n].shape == (cfg["head_dim"],) and abs(float(b[n].mean()) - 1) < 0.01
    assert 0.01 < float(np.std(b["img_q_norm"])) < 0.03
    plain = configs.get_config("flux_small")
    Wp = synth.make_weights(plain, blocks=[0])
    for n, v in Wp["blocks"][0].items():
        if n != "type":
            assert np.array_equal(v, b[n])    # the other tensors are unchanged
    rng = np.random.default_rng(2)
    d, H = 8, 2
    qkv = rng.normal(size=(5, 3 * d)) * 3
    Wb = {"q_norm": np.ones(d // H), "k_norm": np.ones(d // H)}
    q, k = O._qk(qkv, d, Wb, "", H)
    assert np.allclose(np.sqrt(np.mean(q ** 2, axis=-1)), 1.0, atol=1e-6)
    assert np.allclose(np.sqrt(np.mean(k ** 2, axis=-1)), 1.0, atol=1e-6)
    q0, k0 = O._qk(qkv, d, {}, "", H)
    assert np.array_equal(q0, qkv[:, :d].reshape(5, H, -1))


# ---------------------------------------------------------------------------
# UniPC (the sampler of the paper's Wan runs) and the shifted sigma grid
# ---------------------------------------------------------------------------
_S2 = 0.7 ** 2


def _gauss_velocity(x, s):
    """Exact flow-matching velocity for data ~ N(0, 0.7^2) per coordinate."""
    V = (1 - s) ** 2 * _S2 + s ** 2
    return (s - (1 - s) * _S2) / V * x


def _solve(T, shift, vel, x, **kw):
    sig = O.sigma_grid(T, shift)
    if kw.pop("euler", False):
        for i in range(T):
            x = x + (sig[i + 1] - sig[i]) * vel(x, sig[i])
        return x
    u = O.UniPC(sig, **kw)
    for i in range(T):
        x = u.step(i, x, vel(x, sig[i]))
    return x


def test_shifted_sigma_grid():
    assert np.array_equal(O.sigma_grid(8, 1.0), 1 - np.arange(9) / 8)
    g = O.sigma_grid(4, 3.0)
    assert g[0] == 1.0 and g[-1] == 0.0 and np.all(np.diff(g) < 0)
    assert abs(g[2] - 0.75) < 1e-15          # u = 1/2: 3 u / (1 + 2 u)


@pytest.mark.parametrize("shift", [1.0, 5.0])
def test_unipc_first_order_without_corrector_is_euler(shift):
    x0 = np.array([1.3, -0.4, 2.0])
    e = _solve(12, shift, _gauss_velocity, x0, euler=True)
    u = _solve(12, shift, _gauss_velocity, x0, order=1, corrector=False)
    assert np.allclose(u, e, rtol=0, atol=1e-12)


@pytest.mark.parametrize("shift", [1.0, 5.0])
def test_unipc_exact_for_point_mass_data(shift):
    """Data concentrated at one point c: every data prediction is c, every difference
    term vanishes, and the first-order move is the exact flow, so the sampler lands on c."""
    c = np.array([0.3, -1.1])
    vel = lambda x, s: (x - c) / s    # noqa: E731
    for order, corr in ((1, False), (2, True)):
        x = _solve(9, shift, vel, np.array([2.0, 0.5]), order=order, corrector=corr)
        assert np.allclose(x, c, atol=1e-12)


def test_unipc_convergence_orders_on_gaussian_data():
    """The probability-flow ODE of N(0, s^2) data maps x(1) to s x(1).  Euler converges at
    first order; the corrector raises UniPC-1 to second order (UniC adds one order); the
    order-2 predictor-corrector is at least second order and far more accurate."""
    x1 = np.array([1.3, -0.4])
    exact = 0.7 * x1

    def err(T, **kw):
        return float(np.max(np.abs(_solve(T, 1.0, _gauss_velocity, x1, **kw) - exact)))

    e_eu = [err(T, euler=True) for T in (80, 160)]
    e_c1 = [err(T, order=1, corrector=True) for T in (80, 160)]
    e_c2 = [err(T, order=2, corrector=True) for T in (80, 160)]
    assert 1.9 < e_eu[0] / e_eu[1] < 2.1
    assert e_c1[0] / e_c1[1] > 3.4
    assert e_c2[0] / e_c2[1] > 3.6 and e_c2[1] < 0.01 * e_eu[1]


def test_unipc_sampler_budget_T_is_uncached_and_differs_from_euler():
    cfg, W, g, inp = _tiny(grid=(1, 4, 4), n_txt=3)
    cfg = dict(cfg, sampler="unipc", shift=3.0)
    a = O.sample(cfg, W, g, inp, T=6, B=6)
    b = O.sample(cfg, W, g, inp, T=6, B=6, policy="full")
    assert np.array_equal(a["x"], b["x"])
    e = O.sample(dict(cfg, sampler="euler"), W, g, inp, T=6, B=6)
    assert not np.allclose(a["x"], e["x"], atol=1e-6)


# ---------------------------------------------------------------------------
# the network's entry, exit and conditioning pieces
# ---------------------------------------------------------------------------
def test_token_positions_text_at_origin_then_image_row_major():
    cfg = dict(grid=(2, 2, 3), n_txt=2, kind="mmdit")
    pos = O.token_positions(cfg)
    want = [(0, 0, 0)] * 2 + [(f, r, c) for f in range(2) for r in range(2) for c in range(3)]
    assert pos.shape == (14, 3) and [tuple(int(v) for v in p) for p in pos] == want
    wan = O.token_positions(dict(cfg, kind="wan"))  # Wan: no text rows in the sequence
    assert [tuple(int(v) for v in p) for p in wan] == want[2:]


def test_flow_lambda_closed_forms():
    """lambda(sigma) = log((1 - sigma) / sigma): zero at sigma = 1/2, log 4 at 1/5,
    odd under sigma -> 1 - sigma, decreasing, infinite at the ends."""
    assert O.flow_lambda(0.5) == 0.0
    assert abs(O.flow_lambda(0.2) - math.log(4.0)) < 1e-15
    s = np.linspace(0.01, 0.99, 99)
    lam = O.flow_lambda(s)
    assert np.allclose(lam, -O.flow_lambda(1.0 - s), atol=1e-13)
    assert np.all(np.diff(lam) < 0)
    assert O.flow_lambda(1.0) == -np.inf and O.flow_lambda(0.0) == np.inf


def test_patch_embed_selects_weight_columns():
    """x W^T + b with W [d, C]: the unit input e_k gives column k of W plus the bias (a
    transposed weight would give a row)."""
    rng = np.random.default_rng(3)
    C, d = 5, 7
    G = {"pe_w": rng.normal(size=(d, C)), "pe_b": rng.normal(size=d)}
    out = O.patch_embed(G, np.eye(C))
    for k in range(C):
        assert np.allclose(out[k], G["pe_w"][:, k] + G["pe_b"], atol=1e-15)


def test_final_layer_shift_scale_order_and_brute_force():
    """Final layer = Linear(LN-mod(h)) with (shift, scale) = SiLU(vec) W_f^T + b_f split
    shift first.  Scale -1 removes h entirely (output = shift W^T + b), which fails if
    the two halves were swapped; then a scalar-loop evaluation on a tiny case."""
    rng = np.random.default_rng(4)
    d, C, n = 6, 3, 4
    h = rng.normal(size=(n, d)) * 2 + 1
    shift = rng.normal(size=d)
    G = {"fmod_w": np.zeros((2 * d, d)), "fmod_b": np.concatenate([shift, -np.ones(d)]),
         "fin_w": rng.normal(size=(C, d)), "fin_b": rng.normal(size=C)}
    out = O.final_layer(G, rng.normal(size=d), h)
    assert np.allclose(out, np.broadcast_to(shift @ G["fin_w"].T + G["fin_b"], (n, C)), atol=1e-13)
    G["fmod_w"] = rng.normal(size=(2 * d, d)) * 0.3
    G["fmod_b"] = rng.normal(size=2 * d) * 0.3
    vec = rng.normal(size=d)
    sv = [v / (1.0 + math.exp(-v)) for v in vec]
    mod = [sum(G["fmod_w"][o][j] * sv[j] for j in range(d)) + G["fmod_b"][o] for o in range(2 * d)]
    out = O.final_layer(G, vec, h)
    for r in range(n):
        mu = sum(h[r]) / d
        var = sum((h[r][j] - mu) ** 2 for j in range(d)) / d
        y = [(1.0 + mod[d + j]) * (h[r][j] - mu) / math.sqrt(var + 1e-6) + mod[j] for j in range(d)]
        for o in range(C):
            want = sum(G["fin_w"][o][j] * y[j] for j in range(d)) + G["fin_b"][o]
            assert abs(out[r][o] - want) < 1e-12


def test_block_modulation_streams_and_wan_table():
    """SiLU(0) = 0, so a zero conditioning vector leaves each projection's bias: the
    single block's, the image and text streams' own (in that order), and for Wan the
    shared projection's bias plus the block's table."""
    rng = np.random.default_rng(5)
    d = 4
    z = np.zeros(d)
    single = {"type": "single", "mod_w": rng.normal(size=(3 * d, d)), "mod_b": rng.normal(size=3 * d)}
    assert np.array_equal(O.block_modulation({}, {}, single, z), single["mod_b"])
    double = {"type": "double", "img_mod_w": rng.normal(size=(6 * d, d)), "img_mod_b": rng.normal(size=6 * d),
              "txt_mod_w": rng.normal(size=(6 * d, d)), "txt_mod_b": rng.normal(size=6 * d)}
    mi, mt = O.block_modulation({}, {}, double, z)
    assert np.array_equal(mi, double["img_mod_b"]) and np.array_equal(mt, double["txt_mod_b"])
    G = {"tproj_w": rng.normal(size=(6 * d, d)), "tproj_b": rng.normal(size=6 * d)}
    wan = {"type": "wan", "mod_tab": rng.normal(size=6 * d)}
    assert np.allclose(O.block_modulation({}, G, wan, z), G["tproj_b"] + wan["mod_tab"], atol=1e-15)
    # away from zero the projection is W SiLU(vec) + b, W stored [out, in]
    vec = rng.normal(size=d)
    s = vec / (1.0 + np.exp(-vec))
    assert np.allclose(O.block_modulation({}, {}, single, vec),
                       [sum(single["mod_w"][o][j] * s[j] for j in range(d)) + single["mod_b"][o]
                        for o in range(3 * d)], atol=1e-13)


def test_first_modulated_input_reads_the_image_stream_modulation():
    """The signal's observable is block 0's first LN-modulation of the image stream: with
    a double block it takes the image stream's (shift, scale), not the text stream's."""
    rng = np.random.default_rng(6)
    d, n = 4, 5
    blk = {"type": "double", "img_mod_w": np.zeros((6 * d, d)), "img_mod_b": rng.normal(size=6 * d),
           "txt_mod_w": np.zeros((6 * d, d)), "txt_mod_b": rng.normal(size=6 * d)}
    h = rng.normal(size=(n, d))
    got = O.first_modulated_input({"hidden": d}, {}, [blk], rng.normal(size=d), h)
    sh, sc = blk["img_mod_b"][:d], blk["img_mod_b"][d:2 * d]
    for r in range(n):
        mu = sum(h[r]) / d
        var = sum((v - mu) ** 2 for v in h[r]) / d
        for j in range(d):
            want = (1.0 + sc[j]) * (h[r][j] - mu) / math.sqrt(var + 1e-6) + sh[j]
            assert abs(got[r][j] - want) < 1e-12
