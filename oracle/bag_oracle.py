"""fp64 CPU oracle for BAG's cached DiT sampling path.

TEST INFRASTRUCTURE ONLY.  This module is imported by the tests, by the package's smoke
check and by the benchmark's CPU-baseline leg; the product path never calls it.  It
shares no code with the CUDA library: only the seeded input generator (synth.py, which
holds none of the method's arithmetic) feeds both.

What it computes, and from which passage:
  * Budget-exact inference, Algorithm 2 and Sec. 3.2 "Budget-exact inference":
    m_0 = 1 with c = 1; for t >= 1 the gate decides m_t = [sigma(z_t) > tau], then
    "B - c >= T - t => m_t = 1", then "B - c = 0 => m_t = 0"; a full step runs the
    network and refreshes the cache (c += 1), any other step reuses the cached residual.
  * The problem setup of Sec. 3.1: binary mask m with ||m||_1 = B, m_0 = 1; a reused
    step goes "through the standard residual path" (plain residual reuse, Sec. 2).
  * The gate z_t = g_theta(s_bud, s_traj) of Eq. 1, in the 3-input form the build
    targets (remaining-budget fraction, remaining-steps fraction, drift signal) with
    all six scalars of Eq. 3 logged beside it.
  * The trajectory signal: relative L1 change of the observable against the last fully
    computed step (the drift entry of Eq. 3 with the L1 norm); the observable is the
    first block's modulated input by default, or the post-patch-embedding tokens, the
    paper's own observable (Eq. 3), when cfg["observable"] == "embedded".
  * The DiT network evaluated at full steps: adaLN-modulated MMDiT blocks (modulated
    LayerNorm, QKV projection with RoPE, joint attention, output projection, GELU MLP,
    gated residuals).  The paper names the backbones (FLUX.1-dev, Qwen-Image, Wan2.1;
    Sec. 4.1) but not their internals; the block conventions below are the public ones.
  * A flow-matching Euler sampler over sigma_i = 1 - i / T (Sec. 3.1 "T denoising
    steps"; flow matching cited in Sec. 1).

Readings where the paper is silent (also listed in the design notes):
  LayerNorm without affine, eps 1e-6; modulation (1 + scale) * LN(x) + shift; GELU with
  the tanh approximation; attention scale 1/sqrt(head_dim); joint sequence order
  [text; image]; RoPE on interleaved pairs, theta = 10000, per-axis frequencies
  theta^(-2j/d_axis), text tokens at position 0; timestep embedding cos-then-sin of
  1000 * sigma_t over 128 frequencies exp(-ln(10000) j / 128); gate hidden activation
  ReLU; decision on z > logit(tau) (z = logit(tau) reuses); cached residual R = image
  stream after the last block minus the image stream entering the first block;
  text stream not advanced on reused steps.

Precision: everything in float64 except the gate, which is evaluated in float32 in a
fixed operation order (each product and sum rounded separately) because its output is a
binary decision that both implementations must take in the same precision.

Parity pins: see tests/test_oracle_pins.py.  Every function below is pinned by at least
one closed form, invariant, special case or brute-force check there.
"""

import itertools
import math

import numpy as np

TEMB_DIM = 256
ROPE_THETA = 10000.0
LN_EPS = 1e-6
RMS_EPS = 1e-6


# ---------------------------------------------------------------------------
# elementwise pieces
# ---------------------------------------------------------------------------
def silu(x):
    return x / (1.0 + np.exp(-x))


def gelu_tanh(x):
    """GELU, tanh approximation (public FLUX/Wan convention; the paper is silent)."""
    return 0.5 * x * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (x + 0.044715 * x ** 3)))


def layer_norm(x, eps=LN_EPS):
    """Row-wise LayerNorm without affine parameters."""
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps)


def modulate(xn, shift, scale):
    """adaLN modulation (1 + scale) * xn + shift."""
    return xn * (1.0 + scale) + shift


def linear(x, w, b=None):
    """y = x W^T + b with W stored [out, in]."""
    y = x @ w.T
    if b is not None:
        y = y + b
    return y


def timestep_embedding(tval, dim=TEMB_DIM):
    """Sinusoidal embedding of a scalar timestep: [cos(t f_j), sin(t f_j)], j < dim/2."""
    half = dim // 2
    freqs = np.exp(-math.log(10000.0) * np.arange(half, dtype=np.float64) / half)
    args = float(tval) * freqs
    return np.concatenate([np.cos(args), np.sin(args)])


def sigma_grid(T, shift=1.0):
    """Flow-matching noise levels, i = 0..T: u_i = 1 - i/T, optionally time-shifted
    sigma_i = s u_i / (1 + (s - 1) u_i) (s = 1: sigma_i = u_i); sigma_0 = 1, sigma_T = 0."""
    u = 1.0 - np.arange(T + 1, dtype=np.float64) / T
    if shift == 1.0:
        return u
    return shift * u / (1.0 + (shift - 1.0) * u)


# ---------------------------------------------------------------------------
# UniPC (Zhao et al. 2023): the multistep predictor-corrector sampler under which the
# paper caches Wan2.1 (Sec. 4.1), restated for a flow-matching model
# ---------------------------------------------------------------------------
def flow_lambda(sig):
    """Half log-SNR of x = (1 - sigma) x0 + sigma eps: lambda = log((1 - sigma) / sigma)
    (-inf at sigma = 1, +inf at sigma = 0)."""
    sig = np.asarray(sig, np.float64)
    with np.errstate(divide="ignore"):
        return np.log1p(-sig) - np.log(sig)


class UniPC:
    """UniPC in its data-prediction form with B(h) = e^{-h} - 1.

    The model's velocity v at (x_i, sigma_i) gives the data prediction m_i = x_i -
    sigma_i v.  A move from point s to point t (h = lambda_t - lambda_s, alpha = 1 -
    sigma) is

        x_t = (sigma_t / sigma_s) x_s - alpha_t (e^{-h} - 1) m_s
              - alpha_t B(h) sum_k rho_k D_k,     D_k = (m_{k} - m_s) / r_k,
        r_k = (lambda_k - lambda_s) / h,

    over earlier evaluated points k (UniP, the predictor) and, for the corrector UniC,
    also over the new point t itself (r = 1, D = m_t - m_s).  The rho solve
    R rho = b with R[j][k] = r_k^j and b_j = j! psi_{j+1} / B(h), where psi_1 = e^{-h} - 1
    and psi_{j+1} = psi_j / (-h) - 1 / j!.  With one coefficient the fixed value 1/2 is
    used (order-2 predictor, order-1 corrector), UniPC's simple choice.

    Step i: m_i from the model output; if i > 0 the corrector replaces x_i by UniC from
    the previous (corrected) sample with the new m_i (the model is not re-evaluated);
    then the predictor of order p = min(order, i + 1, T - i) (warm-up, first-order last
    step) gives x_{i+1}.  Earlier points with sigma = 1 (lambda = -inf, their terms
    vanish in the limit) are not used."""

    def __init__(self, sig, order=2, corrector=True):
        self.sig = np.asarray(sig, np.float64)
        self.T = len(self.sig) - 1
        self.lam = flow_lambda(self.sig)
        self.order = order
        self.corrector = corrector
        self.ms = {}          # step -> data prediction
        self.x_last = None    # corrected sample of the previous step
        self.hist_last = []   # history points the previous predictor used

    def _move(self, s, t, x_s, hist, m_t=None):
        sig, lam = self.sig, self.lam
        a_t = 1.0 - sig[t]
        a_s = 1.0 - sig[s]
        e_mh = (sig[t] * a_s) / (a_t * sig[s])      # e^{-h}, 0 when sigma_s = 1 or sigma_t = 0
        with np.errstate(divide="ignore"):
            hh = np.log(e_mh)                       # -h
        psi = e_mh - 1.0
        B = psi
        m_s = self.ms[s]
        x_t = (sig[t] / sig[s]) * x_s - a_t * psi * m_s
        rs = [(lam[k] - lam[s]) / (-hh) for k in hist]
        Ds = [(self.ms[k] - m_s) / r for k, r in zip(hist, rs)]
        if m_t is not None:
            rs.append(1.0)
            Ds.append(m_t - m_s)
        n = len(Ds)
        if n == 0:
            return x_t
        if n == 1:
            rho = np.array([0.5])
        else:
            b, fact, p = [], 1.0, psi
            for j in range(1, n + 1):
                p = (p / hh if np.isfinite(hh) else 0.0) - 1.0 / fact
                b.append(fact * p / B)
                fact *= j + 1
            R = np.array([[r ** j for r in rs] for j in range(n)])
            rho = np.linalg.solve(R, np.array(b))
        return x_t - a_t * B * sum(c * D for c, D in zip(rho, Ds))

    def _history(self, s, p):
        """Up to p - 1 earlier evaluated points before s with sigma < 1."""
        return [k for k in range(s - 1, s - p, -1) if k >= 0 and self.sig[k] < 1.0]

    def step(self, i, x, v):
        """Given the sample x_i the model saw and its velocity v_i, return x_{i+1}."""
        m = x - self.sig[i] * v
        if i > 0 and self.corrector:
            self.ms[i] = m
            x = self._move(i - 1, i, self.x_last, self.hist_last, m_t=m)
        self.ms[i] = m
        p = min(self.order, i + 1, self.T - i)
        hist = self._history(i, p)
        x_next = self._move(i, i + 1, x, hist)
        self.x_last = x
        self.hist_last = hist
        return x_next


# ---------------------------------------------------------------------------
# rotary embedding and attention
# ---------------------------------------------------------------------------
def token_positions(cfg):
    """(frame, row, col) of each joint-sequence token: text first at 0, image row-major."""
    f, r, c = cfg["grid"]
    img = np.array([(a, b, e) for a in range(f) for b in range(r) for e in range(c)],
                   dtype=np.float64).reshape(-1, 3)
    if cfg["kind"] == "wan":
        return img
    return np.concatenate([np.zeros((cfg["n_txt"], 3)), img], axis=0)


def rope_angles(pos, axes, theta=ROPE_THETA):
    """Rotation angle of every (token, pair): pairs are laid out axis after axis; pair j
    of an axis of width d_a turns by pos_a * theta^(-2j/d_a)."""
    cols = []
    for a, da in enumerate(axes):
        if da == 0:
            continue
        j = np.arange(da // 2, dtype=np.float64)
        omega = theta ** (-2.0 * j / da)
        cols.append(pos[:, a:a + 1] * omega[None, :])
    return np.concatenate(cols, axis=1)


def apply_rope(x, ang):
    """Rotate interleaved pairs (x[2j], x[2j+1]) of x [N, H, Dh] by ang [N, Dh/2]."""
    c = np.cos(ang)[:, None, :]
    s = np.sin(ang)[:, None, :]
    x0, x1 = x[..., 0::2], x[..., 1::2]
    out = np.empty_like(x)
    out[..., 0::2] = x0 * c - x1 * s
    out[..., 1::2] = x0 * s + x1 * c
    return out


def softmax_rows(s):
    m = s.max(axis=-1, keepdims=True)
    e = np.exp(s - m)
    return e / e.sum(axis=-1, keepdims=True)


def attention(q, k, v, q_rows=None):
    """softmax(q k^T / sqrt(Dh)) v per head.  q [Nq, H, Dh], k, v [Nk, H, Dh].

    q_rows optionally restricts the query rows (the result then has len(q_rows) rows)."""
    if q_rows is not None:
        q = q[q_rows]
    dh = q.shape[-1]
    out = np.empty(q.shape, dtype=np.float64)
    for h in range(q.shape[1]):
        p = softmax_rows(q[:, h, :] @ k[:, h, :].T / math.sqrt(dh))
        out[:, h, :] = p @ v[:, h, :]
    return out


# ---------------------------------------------------------------------------
# blocks
# ---------------------------------------------------------------------------
def _heads(x, H):
    return x.reshape(x.shape[0], H, -1)


def rms_norm_heads(x, w, eps=RMS_EPS):
    """RMSNorm over each head's channels (FLUX / Qwen-Image QK normalisation):
    x [N, H, dh] -> x / sqrt(mean over dh of x^2 + eps) * w, w [dh]."""
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * w


def _qk(qkv, d, W, pre, H):
    """q and k heads of a fused projection [rows, >= 2d] (columns q | k | ...), each
    RMS-normalised per head when the block carries QK-norm scales (pre + 'q_norm',
    pre + 'k_norm'); RoPE comes after."""
    q, k = _heads(qkv[:, :d], H), _heads(qkv[:, d:2 * d], H)
    if pre + "q_norm" in W:
        q = rms_norm_heads(q, W[pre + "q_norm"])
        k = rms_norm_heads(k, W[pre + "k_norm"])
    return q, k


def single_block(h, mod, W, ang, H, rows=None):
    """Single-stream block on the joint sequence h [N, d]; mod = (shift, scale, gate).

    LN-mod -> linear1 (d -> 3d + F: q, k, v, mlp) -> RoPE(q, k) -> attention;
    GELU(mlp); linear2 on [attn | GELU(mlp)] -> gated residual.
    rows: compute the output only at these rows (the others are not returned)."""
    d = h.shape[1]
    shift, scale, gate = mod[:d], mod[d:2 * d], mod[2 * d:3 * d]
    xn = modulate(layer_norm(h), shift, scale)
    w1, b1 = W["lin1_w"], W["lin1_b"]
    qkv = linear(xn, w1[:3 * d], b1[:3 * d])
    q, k = _qk(qkv, d, W, "", H)
    q, k = apply_rope(q, ang), apply_rope(k, ang)
    v = _heads(qkv[:, 2 * d:], H)
    sel = slice(None) if rows is None else rows
    a = attention(q, k, v, q_rows=rows).reshape(-1, d)
    mlp = gelu_tanh(linear(xn[sel], w1[3 * d:], b1[3 * d:]))
    o = linear(np.concatenate([a, mlp], axis=1), W["lin2_w"], W["lin2_b"])
    return h[sel] + gate * o


def _mlp(x, wu, bu, wd, bd):
    return linear(gelu_tanh(linear(x, wu, bu)), wd, bd)


def double_block(img, txt, mod_img, mod_txt, W, ang, H, rows=None):
    """Double-stream (MMDiT) block: separate weights per stream, joint attention over
    [txt; img].  mod_* = (shift1, scale1, gate1, shift2, scale2, gate2).

    rows: optional joint-sequence rows (text first) at which to evaluate the outputs;
    then the return value is the joint output [len(rows), d] at those rows only."""
    d = img.shape[1]
    nx = txt.shape[0]

    def chunks(m):
        return [m[i * d:(i + 1) * d] for i in range(6)]

    mi, mt = chunks(mod_img), chunks(mod_txt)
    qkv_i = linear(modulate(layer_norm(img), mi[0], mi[1]), W["img_qkv_w"], W["img_qkv_b"])
    qkv_t = linear(modulate(layer_norm(txt), mt[0], mt[1]), W["txt_qkv_w"], W["txt_qkv_b"])
    qkv = np.concatenate([qkv_t, qkv_i], axis=0)
    (q_t, k_t), (q_i, k_i) = _qk(qkv_t, d, W, "txt_", H), _qk(qkv_i, d, W, "img_", H)
    q = apply_rope(np.concatenate([q_t, q_i], axis=0), ang)
    k = apply_rope(np.concatenate([k_t, k_i], axis=0), ang)
    v = _heads(qkv[:, 2 * d:], H)
    if rows is not None:
        rows = np.asarray(rows)
        a = attention(q, k, v, q_rows=rows).reshape(-1, d)
        hj = np.concatenate([txt, img], axis=0)[rows]
        out = np.empty_like(hj)
        for sel, pre, m in ((rows < nx, "txt", mt), (rows >= nx, "img", mi)):
            if not sel.any():
                continue
            x = hj[sel] + m[2] * linear(a[sel], W[pre + "_proj_w"], W[pre + "_proj_b"])
            out[sel] = x + m[5] * _mlp(modulate(layer_norm(x), m[3], m[4]), W[pre + "_up_w"],
                                       W[pre + "_up_b"], W[pre + "_down_w"], W[pre + "_down_b"])
        return out
    a = attention(q, k, v).reshape(-1, d)
    a_t, a_i = a[:nx], a[nx:]
    img = img + mi[2] * linear(a_i, W["img_proj_w"], W["img_proj_b"])
    txt = txt + mt[2] * linear(a_t, W["txt_proj_w"], W["txt_proj_b"])
    img = img + mi[5] * _mlp(modulate(layer_norm(img), mi[3], mi[4]),
                             W["img_up_w"], W["img_up_b"], W["img_down_w"], W["img_down_b"])
    txt = txt + mt[5] * _mlp(modulate(layer_norm(txt), mt[3], mt[4]),
                             W["txt_up_w"], W["txt_up_b"], W["txt_down_w"], W["txt_down_b"])
    return img, txt


def wan_block(x, ctx, e, W, ang, H, rows=None):
    """Wan-style block: modulated self-attention with 3D RoPE, cross-attention to the
    text context (plain LayerNorm on the query side, no gate), modulated GELU FFN.
    e = (shift1, scale1, gate1, shift2, scale2, gate2).
    rows: optional image rows at which to evaluate (then only those rows are returned)."""
    d = x.shape[1]
    ch = [e[i * d:(i + 1) * d] for i in range(6)]
    qkv = linear(modulate(layer_norm(x), ch[0], ch[1]), W["sa_qkv_w"], W["sa_qkv_b"])
    q = apply_rope(_heads(qkv[:, :d], H), ang)
    k = apply_rope(_heads(qkv[:, d:2 * d], H), ang)
    v = _heads(qkv[:, 2 * d:], H)
    if rows is not None:
        rows = np.asarray(rows)
        x = x[rows]
    x = x + ch[2] * linear(attention(q, k, v, q_rows=rows).reshape(-1, d), W["sa_o_w"], W["sa_o_b"])
    qc = _heads(linear(layer_norm(x), W["ca_q_w"], W["ca_q_b"]), H)
    kv = linear(ctx, W["ca_kv_w"], W["ca_kv_b"])
    kc, vc = _heads(kv[:, :d], H), _heads(kv[:, d:], H)
    x = x + linear(attention(qc, kc, vc).reshape(-1, d), W["ca_o_w"], W["ca_o_b"])
    x = x + ch[5] * _mlp(modulate(layer_norm(x), ch[3], ch[4]),
                         W["ffn_up_w"], W["ffn_up_b"], W["ffn_down_w"], W["ffn_down_b"])
    return x


# ---------------------------------------------------------------------------
# network pieces around the stack
# ---------------------------------------------------------------------------
def conditioning(cfg, G, sigma, pooled):
    """vec = MLP(sinusoid(1000 sigma)) (+ pooled text vector except for Wan)."""
    e = timestep_embedding(1000.0 * sigma)
    temb = linear(silu(linear(e, G["t1_w"], G["t1_b"])), G["t2_w"], G["t2_b"])
    if cfg["kind"] == "wan":
        return temb
    return temb + pooled


def block_modulation(cfg, G, blk, vec):
    """Per-block modulation vectors from the conditioning vector."""
    if blk["type"] == "single":
        return linear(silu(vec), blk["mod_w"], blk["mod_b"])
    if blk["type"] == "double":
        return (linear(silu(vec), blk["img_mod_w"], blk["img_mod_b"]),
                linear(silu(vec), blk["txt_mod_w"], blk["txt_mod_b"]))
    # Wan: one shared projection of the time embedding plus a per-block table
    return linear(silu(vec), G["tproj_w"], G["tproj_b"]) + blk["mod_tab"]


def first_modulated_input(cfg, G, blocks, vec, h_img):
    """Image-stream input of the first block after its first LN-modulation: the
    observable the trajectory signal reads."""
    d = cfg["hidden"]
    mod = block_modulation(cfg, G, blocks[0], vec)
    if blocks[0]["type"] == "double":
        mod = mod[0]
    return modulate(layer_norm(h_img), mod[:d], mod[d:2 * d])


def patch_embed(G, x):
    return linear(x, G["pe_w"], G["pe_b"])


def observable(cfg, G, blocks, vec, h_in):
    """What the trajectory signal of Eq. 3 reads at a step.  'embedded': the
    post-patch-embedding token tensor x_t itself, the paper's choice (Eq. 3 and the
    paragraph after it; under guidance it is shared by both branches).  'modulated'
    (default): the first block's modulated input on the image stream."""
    if cfg.get("observable", "modulated") == "embedded":
        return h_in
    return first_modulated_input(cfg, G, blocks, vec, h_in)


def run_stack(cfg, G, blocks, vec, h_img, txt):
    """Full network stack on the image stream h_img [N_i, d] with text txt; returns the
    image stream after the last block."""
    H = cfg["heads"]
    pos = token_positions(cfg)
    ang = rope_angles(pos, cfg["rope_axes"])
    if cfg["kind"] == "wan":
        x = h_img
        for blk in blocks:
            x = wan_block(x, txt, block_modulation(cfg, G, blk, vec), blk, ang, H)
        return x
    img, tx = h_img, txt
    nx = txt.shape[0]
    singles_started = False
    hj = None
    for blk in blocks:
        mod = block_modulation(cfg, G, blk, vec)
        if blk["type"] == "double":
            assert not singles_started
            img, tx = double_block(img, tx, mod[0], mod[1], blk, ang, H)
        else:
            if not singles_started:
                hj = np.concatenate([tx, img], axis=0)
                singles_started = True
            hj = single_block(hj, mod, blk, ang, H)
    if singles_started:
        img = hj[nx:]
    return img


def final_layer(G, vec, h_img):
    d = h_img.shape[1]
    mod = linear(silu(vec), G["fmod_w"], G["fmod_b"])
    return linear(modulate(layer_norm(h_img), mod[:d], mod[d:]), G["fin_w"], G["fin_b"])


def rel_l1(a, b):
    """Relative L1 change sum|a - b| / sum|b| (the drift entry of Eq. 3, L1 norm)."""
    return float(np.abs(a - b).sum() / np.abs(b).sum())


# ---------------------------------------------------------------------------
# gate and pacing (Eq. 1, Eq. 3, Algorithm 2)
# ---------------------------------------------------------------------------
F32 = np.float32


def gate_threshold(tau):
    """Decision threshold on the logit: sigma(z) > tau  <=>  z > log(tau / (1 - tau))."""
    return F32(math.log(tau / (1.0 - tau)))


def gate_features(B, T, c, t, drift):
    """The three gate inputs at step t with c evaluations already spent: remaining-budget
    fraction (B - c)/B (Eq. 3), remaining-steps fraction (T - t)/T, drift signal."""
    return [F32(B - c) / F32(B), F32(T - t) / F32(T), F32(drift)]


def gate_logit(f, g):
    """z = w2 . ReLU(W1 ((f - mu) / sd) + b1) + b2 in float32, fixed order: every product
    and every sum rounded on its own, inputs visited in index order."""
    fz = [(F32(f[i]) - F32(g["mu"][i])) / F32(g["sd"][i]) for i in range(len(f))]
    w1, b1, w2, b2 = g["w1"], g["b1"], g["w2"], g["b2"]
    z = F32(b2[0])
    for j in range(w1.shape[0]):
        hj = F32(b1[j])
        for i in range(len(fz)):
            hj = F32(hj + F32(F32(w1[j, i]) * fz[i]))
        if not hj > F32(0.0):
            hj = F32(0.0)
        z = F32(z + F32(F32(w2[j]) * hj))
    return z


def gate_features6(B, T, c, t, t_last, drift, step):
    """The six scalars of Eq. 3 in float32: s_bud = [B/T, (B-c)/B, (B-c)/(T-t)],
    s_traj = [t - t_last, drift since the last full step, step-to-step change]."""
    return [F32(B) / F32(T), F32(B - c) / F32(B), F32(B - c) / F32(T - t),
            F32(t - t_last), F32(drift), F32(step)]


def _dense32(x, W, b, relu):
    """fp32 dense layer in a fixed order: out_j = b_j + sum_i W[j, i] x_i, inputs in index
    order, every product and sum rounded on its own; optional ReLU."""
    out = []
    for j in range(W.shape[0]):
        h = F32(b[j])
        for i in range(len(x)):
            h = F32(h + F32(F32(W[j, i]) * x[i]))
        if relu and not h > F32(0.0):
            h = F32(0.0)
        out.append(h)
    return out


def gate_logit6(f, g):
    """The paper's six-input gates (App. A.2) on z-scored inputs, fp32, ReLU hidden
    activations: "flux6" one MLP 6-8-8-32-1; "wan6" budget branch 3-8-8 and trajectory
    branch 3-8-8, concatenated [budget, trajectory], fused by 16-32-1."""
    fz = [(F32(f[i]) - F32(g["mu"][i])) / F32(g["sd"][i]) for i in range(6)]
    L = list(zip(g["W"], g["b"]))
    if g["kind"] == "flux6":
        h = fz
        for k, (W, b) in enumerate(L):
            h = _dense32(h, W, b, relu=k < len(L) - 1)
        return h[0]
    hb = _dense32(_dense32(fz[:3], *L[0], relu=True), *L[1], relu=True)
    ht = _dense32(_dense32(fz[3:], *L[2], relu=True), *L[3], relu=True)
    h = _dense32(hb + ht, *L[4], relu=True)
    return _dense32(h, *L[5], relu=False)[0]


# ---------------------------------------------------------------------------
# training side (Algorithm 1): Eq. 2's reference schedule and Eq. 4's loss
# ---------------------------------------------------------------------------
def all_masks(B, T):
    """Every schedule with ||m||_1 = B and m_0 = 1 (Sec. 3.1), in lexicographic order of
    the computed steps."""
    for rest in itertools.combinations(range(1, T), B - 1):
        m = [0] * T
        m[0] = 1
        for t in rest:
            m[t] = 1
        yield m


def reference_by_enumeration(distance, B, T):
    """Eq. 2 by brute force: the mask minimising distance(mask) over all matched-NFE
    masks (the first one on ties).  Returns (mask, distance)."""
    best, best_d = None, math.inf
    for m in all_masks(B, T):
        dm = distance(m)
        if dm < best_d:
            best, best_d = m, dm
    return best, best_d


def gate_forward64(g, xz):
    """Gate logit in float64 on already z-scored inputs xz [n, k] (rows = examples):
    the same architectures as gate_logit / gate_logit6 without fp32 rounding."""
    xz = np.asarray(xz, np.float64)
    relu = lambda v: np.maximum(v, 0.0)   # noqa: E731
    if g.get("kind", "mlp3") == "mlp3":
        return relu(xz @ np.asarray(g["w1"], np.float64).T + g["b1"]) @ np.asarray(g["w2"], np.float64) + g["b2"][0]
    L = [(np.asarray(W, np.float64), np.asarray(b, np.float64)) for W, b in zip(g["W"], g["b"])]
    if g["kind"] == "flux6":
        h = xz
        for k, (W, b) in enumerate(L):
            h = h @ W.T + b
            if k < len(L) - 1:
                h = relu(h)
        return h[:, 0]
    hb = relu(relu(xz[:, :3] @ L[0][0].T + L[0][1]) @ L[1][0].T + L[1][1])
    ht = relu(relu(xz[:, 3:] @ L[2][0].T + L[2][1]) @ L[3][0].T + L[3][1])
    h = relu(np.concatenate([hb, ht], axis=1) @ L[4][0].T + L[4][1])
    return (h @ L[5][0].T + L[5][1])[:, 0]


def zscore_stats(X):
    """Per-input mean and standard deviation of the training examples (Sec. 3.2: the
    inputs are z-scored); a constant input gets sd = 1."""
    X = np.asarray(X, np.float64)
    mu, sd = X.mean(axis=0), X.std(axis=0)
    return mu, np.where(sd > 0, sd, 1.0)


def distillation_loss(g, X, y):
    """Eq. 4 (divided by |D|), class-balanced: mean over examples of w_i BCE(sigma(z_i), y_i), z_i the gate
    on (x_i - mu) / sd, positives weighted by the negative-to-positive count ratio
    (App. A.2), negatives by 1.  float64."""
    X, y = np.asarray(X, np.float64), np.asarray(y, np.float64)
    z = gate_forward64(g, (X - g["mu"]) / g["sd"])
    n_pos = float(y.sum())
    w_pos = (len(y) - n_pos) / n_pos if n_pos > 0 else 1.0
    # BCE(sigma(z), y) = softplus(z) - y z, written stably
    sp = np.maximum(z, 0.0) + np.log1p(np.exp(-np.abs(z)))
    per = np.where(y > 0.5, w_pos * (sp - z), sp)
    return float(per.mean())


def pace(gate_bit, B, T, c, t):
    """Algorithm 2's forced rules applied to the gate's bit at step t >= 1."""
    m = 1 if gate_bit else 0
    if B - c >= T - t:
        m = 1        # spend the remainder
    if B - c == 0:
        m = 0        # budget exhausted
    return m


def static_uniform_schedule(B, T):
    """Open-loop schedule mu(B, T) of Sec. 3.1's static paradigm, evenly spaced: the
    steps floor(i * T / B), i = 0 .. B-1 (step 0 included, B distinct steps)."""
    m = [0] * T
    for i in range(B):
        m[(i * T) // B] = 1
    return m


def threshold_decision(drift, delta):
    """Online threshold paradigm of Sec. 3.1: m_t = [q_t > delta] with q_t the drift
    since the last full step, compared in fp32; no budget enters the decision."""
    return 1 if F32(drift) > F32(delta) else 0


def schedule_from_gate_bits(bits, B, T):
    """Mask produced by Algorithm 2 from a sequence of raw gate bits (bits[0] unused)."""
    m = [1]
    c = 1
    for t in range(1, T):
        mt = pace(bits[t], B, T, c, t)
        m.append(mt)
        c += mt
    return m


# ---------------------------------------------------------------------------
# the sampler (Algorithm 2 with the network, the signal and the residual cache)
# ---------------------------------------------------------------------------
def to64(W):
    """Upcast a weight tree (as produced by the seeded generator) to float64."""
    out = {"global": {k: np.asarray(v, np.float64) for k, v in W["global"].items()},
           "blocks": []}
    for blk in W["blocks"]:
        out["blocks"].append(None if blk is None else
                             {k: (v if k == "type" else np.asarray(v, np.float64))
                              for k, v in blk.items()})
    return out


def sample(cfg, W, gate, inputs, T, B, tau=0.5, policy="bag", drift_override=None,
           step_override=None, guidance=None):
    """One sample of T sampler steps under Algorithm 2: Euler on the (optionally shifted)
    sigma grid, or UniPC of order 2 when cfg["sampler"] == "unipc" (cfg["shift"]: the
    grid's time shift, default 1).

    policy         'bag' (gate + pacing), 'full' (uncached: every step computes),
                   'uniform' (static evenly spaced schedule of B steps), ('threshold', d)
                   (online rule drift > d, realised NFE not fixed), or a list of T mask
                   bits to follow (a static schedule).
    drift_override optional per-step drift values (index t) to feed the gate instead of
                   the oracle's own; used to take the decision on another
                   implementation's logged gate inputs.
    step_override  likewise for the step-to-step change (six-input gates).
    guidance       classifier-free guidance scale g (None: no guidance).  Then inputs
                   also holds "txt_u" / "pooled_u" (the unconditional branch), both
                   branches share one mask (a step is computed for both or reused for
                   both, App. A.1), each keeps its own cached residual, the signal is
                   read on the conditional branch (Eq. 3), and v = v_u + g (v_c - v_u).
    The gate is the 3-input MLP unless gate["kind"] names a six-input gate.
    Returns dict(x=final latent, mask, log=[per-step dict]).
    """
    if not (1 <= B <= T):
        raise ValueError("need 1 <= B <= T")
    W = to64(W)
    G, blocks = W["global"], W["blocks"]
    x = np.asarray(inputs["x"], np.float64)
    txt = np.asarray(inputs["txt"], np.float64)
    pooled = np.asarray(inputs["pooled"], np.float64)
    if guidance is not None:
        txt_u = np.asarray(inputs["txt_u"], np.float64)
        pooled_u = np.asarray(inputs["pooled_u"], np.float64)
        R_u = None
    sig = sigma_grid(T, cfg.get("shift", 1.0))
    solver = UniPC(sig) if cfg.get("sampler", "euler") == "unipc" else None
    thr = gate_threshold(tau)
    c = 0
    t_last = -1
    R = m_last = m_prev = None
    mask, log = [], []
    for t in range(T):
        vec = conditioning(cfg, G, sig[t], pooled)
        h_in = patch_embed(G, x)
        m_t = observable(cfg, G, blocks, vec, h_in)
        rec = {"t": t, "c_before": c}
        if t == 0:
            full = 1
        else:
            drift = rel_l1(m_t, m_last)
            rec["drift"] = drift
            # the six scalars of Eq. 3, logged
            rec["s_bud"] = [B / T, (B - c) / B, (B - c) / (T - t)]
            rec["s_traj"] = [t - t_last, drift, rel_l1(m_t, m_prev)]
            used = drift if drift_override is None else drift_override[t]
            if gate.get("kind", "mlp3") == "mlp3":
                f = gate_features(B, T, c, t, used)
                z = gate_logit(f, gate)
            else:
                step = rec["s_traj"][2] if step_override is None else step_override[t]
                f = gate_features6(B, T, c, t, t_last, used, step)
                z = gate_logit6(f, gate)
            rec["features"] = [float(v) for v in f]
            rec["z"] = float(z)
            gbit = 1 if z > thr else 0
            if policy == "bag":
                full = pace(gbit, B, T, c, t)
            elif policy == "full":
                full = 1
            elif policy == "uniform":
                full = static_uniform_schedule(B, T)[t]
            elif isinstance(policy, tuple) and policy[0] == "threshold":
                full = threshold_decision(used, policy[1])
            else:
                full = int(policy[t])
        rec["full"] = full
        if guidance is not None:
            vec_u = conditioning(cfg, G, sig[t], pooled_u)
        if full:
            h_out = run_stack(cfg, G, blocks, vec, h_in, txt)
            R = h_out - h_in
            if guidance is not None:
                h_out_u = run_stack(cfg, G, blocks, vec_u, h_in, txt_u)
                R_u = h_out_u - h_in
            m_last = m_t
            t_last = t
            c += 1
        else:
            h_out = h_in + R
            if guidance is not None:
                h_out_u = h_in + R_u
        m_prev = m_t
        v = final_layer(G, vec, h_out)
        if guidance is not None:
            v_u = final_layer(G, vec_u, h_out_u)
            v = v_u + guidance * (v - v_u)
        if solver is not None:
            x = solver.step(t, x, v)
        else:
            x = x + (sig[t + 1] - sig[t]) * v
        mask.append(full)
        log.append(rec)
    return {"x": x, "mask": mask, "log": log, "nfe": c}


def forward_block(cfg, W, block_index, h_joint, vec, rows=None, txt=None):
    """One block of the stack applied to a given stream: the joint [txt; img] sequence
    (text rows first) for single- and double-stream blocks, the image stream for Wan
    blocks (txt = the cross-attention context).  rows: evaluate only those rows."""
    W = to64(W)
    G, blk = W["global"], W["blocks"][block_index]
    H = cfg["heads"]
    ang = rope_angles(token_positions(cfg), cfg["rope_axes"])
    mod = block_modulation(cfg, G, blk, vec)
    if blk["type"] == "single":
        return single_block(h_joint, mod, blk, ang, H, rows=rows)
    if blk["type"] == "double":
        nx = cfg["n_txt"]
        out = double_block(h_joint[nx:], h_joint[:nx], mod[0], mod[1], blk, ang, H, rows=rows)
        if rows is None:
            return np.concatenate([out[1], out[0]], axis=0)
        return out
    return wan_block(h_joint, txt, mod, blk, ang, H, rows=rows)
