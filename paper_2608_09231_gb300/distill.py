"""The offline side of BAG at toy scale: the matched-NFE reference search of Eq. 2
(App. A.1, with the mean squared error to the full-compute output as the distance D in
place of LPIPS) and the gate's supervised distillation (Algorithm 1, Eq. 4).

Rollouts run through the CUDA library: one context samples the same inputs under
caller-given masks (BAG_POLICY_MASK), and the per-step states of Eq. 3 come from the
step log the gate kernel writes.  The search loop and the training loop are host code;
they run once per backbone, never at deployment.
"""

import math

import numpy as np

from . import bag, synth

# Gate inputs inside a logged step record (bag.h, BAG_LOG_FLOATS layout).  Six-input
# gates read Eq. 3's scalars in the paper's order [B/T, (B-c)/B, (B-c)/(T-t), t - t_last,
# drift, step change]; the three-input gate reads [(B-c)/B, (T-t)/T, drift].
LOG_COLS = {"mlp3": [0, 1, 2], "flux6": [8, 9, 10, 7, 2, 13], "wan6": [8, 9, 10, 7, 2, 13]}


# ---------------------------------------------------------------------------
# masks
# ---------------------------------------------------------------------------
def _check(mask, B, T):
    if len(mask) != T or int(sum(mask)) != B or mask[0] != 1:
        raise ValueError(f"not a matched-NFE mask for B={B}, T={T}: {mask}")


def uniform_mask(B, T):
    """B computed steps evenly spaced, floor(i T / B) (the static paradigm, Sec. 3.1)."""
    m = [0] * T
    for i in range(B):
        m[i * T // B] = 1
    return m


def front_loaded_mask(B, T):
    """A start that spends the budget early: steps 0 .. B-1."""
    return [1] * B + [0] * (T - B)


def insert_steps(mask, B, rng=None):
    """Raise a lower budget's mask to B computed steps by computing some of its reused
    steps: evenly spaced among them (rng None) or at random (App. A.1's starts at higher
    budgets)."""
    m = list(mask)
    free = [t for t in range(1, len(m)) if not m[t]]
    extra = B - sum(m)
    if extra < 0 or extra > len(free):
        raise ValueError("cannot insert that many steps")
    if extra == 0:
        return m
    if rng is None:
        pick = [free[(2 * i + 1) * len(free) // (2 * extra)] for i in range(extra)]
    else:
        pick = list(rng.choice(free, size=extra, replace=False))
    for t in pick:
        m[int(t)] = 1
    return m


def _moves(mask):
    """(shifts, relocations): masks one move away (App. A.1: a move shifts or relocates
    one computed step) - a computed step t >= 1 moved to the reused step t - 1 or t + 1,
    or to any other reused step.  Step 0 stays computed."""
    T = len(mask)
    on = [t for t in range(1, T) if mask[t]]
    off = [t for t in range(1, T) if not mask[t]]
    shifts, relocs = [], []
    for a in on:
        for b in off:
            m = list(mask)
            m[a], m[b] = 0, 1
            (shifts if abs(a - b) == 1 else relocs).append(m)
    return shifts, relocs


def neighbors(mask):
    """Every mask one move away, the shifts first (each mask once)."""
    shifts, relocs = _moves(mask)
    return shifts + relocs


# ---------------------------------------------------------------------------
# search (Eq. 2, App. A.1)
# ---------------------------------------------------------------------------
def local_search(distance, B, T, starts, rng=None, anneal_steps=0, temp0=None, cooling=0.9,
                 max_evals=None):
    """Multi-start local search for Eq. 2's reference mask.

    distance(mask) -> float is D(x_T(m), x_T(1)); every evaluated mask's value is cached
    (a rollout is deterministic given its mask).  With anneal_steps > 0 a short
    simulated-annealing walk runs from each of the three best starts (random moves,
    Metropolis acceptance, geometric cooling from temp0, default a tenth of the best
    start's distance); then greedy refinement takes the first improving move (shifts
    before relocations, otherwise in rng order) until none improves, or until max_evals
    distinct masks have been rolled out.  Returns dict(mask, distance, evals)."""
    rng = np.random.default_rng(0) if rng is None else rng
    cache = {}

    def D(m):
        k = tuple(m)
        if k not in cache:
            cache[k] = float(distance(list(m)))
        return cache[k]

    def budget_left():
        return max_evals is None or len(cache) < max_evals

    for s in starts:
        _check(s, B, T)
    ranked = sorted((list(s) for s in starts), key=D)
    best = ranked[0]
    if anneal_steps > 0 and B < T:
        for s in ranked[:3]:
            cur, dcur = s, D(s)
            temp = temp0 if temp0 is not None else 0.1 * max(D(ranked[0]), 1e-30)
            for _ in range(anneal_steps):
                if not budget_left():
                    break
                nb = neighbors(cur)
                cand = nb[int(rng.integers(len(nb)))]
                dc = D(cand)
                if dc < dcur or rng.random() < math.exp(-(dc - dcur) / max(temp, 1e-300)):
                    cur, dcur = cand, dc
                if dcur < D(best):
                    best = cur
                temp *= cooling
    improved = True
    while improved and budget_left():
        improved = False
        shifts, relocs = _moves(best)
        for m in shifts + [relocs[i] for i in rng.permutation(len(relocs))]:
            if not budget_left():
                break
            if D(m) < D(best):
                best, improved = m, True
                break
    return {"mask": best, "distance": D(best), "evals": len(cache)}


# ---------------------------------------------------------------------------
# rollouts through the CUDA library
# ---------------------------------------------------------------------------
class Rollouts:
    """Samples of one fixed input (a "prompt" and its seed) through a context, under
    caller-given masks: the target x_T(1), the distance of Eq. 2 (mean squared error to
    the target) and the logged per-step states along a rollout."""

    def __init__(self, ctx, inputs):
        import torch

        cfg = ctx.cfg
        self.ctx = ctx
        self.T = ctx.T
        self.x0 = torch.from_numpy(np.ascontiguousarray(inputs["x"], np.float32)).cuda()
        txt = torch.from_numpy(np.ascontiguousarray(inputs["txt"], np.float32)).cuda()
        if cfg["dtype"] == "bf16":
            txt = txt.to(torch.bfloat16)
        self.cond = [txt, torch.from_numpy(np.ascontiguousarray(inputs["pooled"], np.float32)).cuda()]
        if cfg.get("guidance") is not None:
            txt_u = torch.from_numpy(np.ascontiguousarray(inputs["txt_u"], np.float32)).cuda()
            self.cond += [txt_u.to(txt.dtype),
                          torch.from_numpy(np.ascontiguousarray(inputs["pooled_u"], np.float32)).cuda()]
        self.x = torch.empty_like(self.x0)
        self.rollouts = 0
        self._target = None

    def run(self, mask):
        """x_T under `mask` (its NFE becomes the context's budget); returns (x_T, log)."""
        import torch

        B = int(sum(mask))
        _check(list(mask), B, self.T)
        if self.ctx.B != B:
            self.ctx.set_budget(B)
        self.ctx.set_policy(bag.POLICY_MASK, np.asarray(mask, np.uint8))
        self.ctx.reset()
        self.x.copy_(self.x0)
        _, log, nfe = self.ctx.run(self.x, *self.cond)
        torch.cuda.synchronize()
        self.rollouts += 1
        if nfe != B:
            raise RuntimeError(f"rollout spent {nfe} evaluations, mask has {B}")
        return self.x.cpu().numpy().astype(np.float64), log

    def target(self):
        """The full-compute output x_T(1) (cached)."""
        if self._target is None:
            self._target = self.run([1] * self.T)[0]
        return self._target

    def distance(self, mask):
        """Eq. 2's D with the mean squared error: mean (x_T(m) - x_T(1))^2."""
        x, _ = self.run(mask)
        return float(np.mean((x - self.target()) ** 2))


def examples_from_log(log, mask, kind="flux6"):
    """Algorithm 1's per-step examples along one rollout: the gate inputs the step log
    recorded at t >= 1 and the reference decision m_t."""
    X = np.asarray(log, np.float64)[1:, LOG_COLS[kind]]
    y = np.asarray(mask, np.float64)[1:]
    return X, y


def reference_examples(ctx, inputs_list, budgets, kind="flux6", anneal_steps=20, seed=0,
                       max_evals=None):
    """The two loops of Algorithm 1: for every input and budget, search the reference mask
    (starts: uniform, front-loaded, and the next lower budget's reference with steps
    inserted evenly), then record the states along its rollout.  Returns (X, y, cells),
    cells a list of dict(input, B, mask, distance, evals)."""
    rng = np.random.default_rng(seed)
    T = ctx.T
    Xs, ys, cells = [], [], []
    for ii, inp in enumerate(inputs_list):
        ro = Rollouts(ctx, inp)
        ro.target()
        prev = None
        for B in sorted(budgets):
            starts = [uniform_mask(B, T), front_loaded_mask(B, T)]
            if prev is not None:
                starts.append(insert_steps(prev, B))
            res = local_search(ro.distance, B, T, starts, rng=rng, anneal_steps=anneal_steps,
                               max_evals=max_evals)
            _, log = ro.run(res["mask"])
            X, y = examples_from_log(log, res["mask"], kind)
            Xs.append(X)
            ys.append(y)
            cells.append(dict(input=ii, B=B, mask=res["mask"], distance=res["distance"],
                              evals=res["evals"]))
            prev = res["mask"]
    return np.concatenate(Xs), np.concatenate(ys), cells


# ---------------------------------------------------------------------------
# distillation (Eq. 4)
# ---------------------------------------------------------------------------
def auc(scores, y):
    """Area under the ROC curve (probability that a positive outranks a negative; ties
    count one half)."""
    scores, y = np.asarray(scores, np.float64), np.asarray(y) > 0.5
    pos, neg = scores[y], scores[~y]
    if len(pos) == 0 or len(neg) == 0:
        return float("nan")
    order = np.argsort(np.concatenate([pos, neg]), kind="mergesort")
    allv = np.concatenate([pos, neg])[order]
    ranks = np.empty(len(allv))
    i = 0
    while i < len(allv):      # average ranks over ties
        j = i
        while j + 1 < len(allv) and allv[j + 1] == allv[i]:
            j += 1
        ranks[i:j + 1] = 0.5 * (i + j) + 1
        i = j + 1
    r = np.empty(len(allv))
    r[order] = ranks
    return float((r[:len(pos)].sum() - len(pos) * (len(pos) + 1) / 2) / (len(pos) * len(neg)))


def fit_gate(X, y, kind="flux6", epochs=300, lr=1e-3, weight_decay=1e-4, batch=8192, seed=0,
             gate_seed=None):
    """Fit the gate on Algorithm 1's examples: inputs z-scored with the training set's
    statistics, class-balanced BCE on the logit (positives weighted by the negative-to-
    positive ratio, Eq. 4 and App. A.2), AdamW.  Starts from the seeded gate of that
    kind (gate_seed, default seed).  Returns (gate, history): gate in the seeded
    generator's layout (loadable with Context.load_gate via synth.gate_flat), history a
    list of dict(epoch, loss, auc) per epoch (loss = Eq. 4 divided by |D|)."""
    import torch

    X = np.asarray(X, np.float64)
    y = np.asarray(y, np.float64)
    mu = X.mean(axis=0)
    sd = X.std(axis=0)
    sd = np.where(sd > 0, sd, 1.0)
    g0 = synth.make_gate_any(seed if gate_seed is None else gate_seed, kind)
    if kind == "mlp3":
        Ws, bs = [g0["w1"], g0["w2"][None, :]], [g0["b1"], g0["b2"]]
    else:
        Ws, bs = g0["W"], g0["b"]
    params = []
    for W, b in zip(Ws, bs):
        params.append(torch.tensor(np.asarray(W, np.float32), requires_grad=True))
        params.append(torch.tensor(np.asarray(b, np.float32), requires_grad=True))
    xz = torch.tensor(((X - mu) / sd).astype(np.float32))
    yt = torch.tensor(y.astype(np.float32))
    n_pos = float(y.sum())
    pos_weight = torch.tensor((len(y) - n_pos) / n_pos if n_pos > 0 else 1.0)

    def forward(inp):
        L = [(params[2 * i], params[2 * i + 1]) for i in range(len(params) // 2)]
        if kind == "wan6":
            hb = torch.relu(torch.relu(inp[:, :3] @ L[0][0].T + L[0][1]) @ L[1][0].T + L[1][1])
            ht = torch.relu(torch.relu(inp[:, 3:] @ L[2][0].T + L[2][1]) @ L[3][0].T + L[3][1])
            h = torch.relu(torch.cat([hb, ht], dim=1) @ L[4][0].T + L[4][1])
            return (h @ L[5][0].T + L[5][1])[:, 0]
        h = inp
        for k, (W, b) in enumerate(L):
            h = h @ W.T + b
            if k < len(L) - 1:
                h = torch.relu(h)
        return h[:, 0]

    def loss_fn(z, t):
        return torch.nn.functional.binary_cross_entropy_with_logits(z, t, pos_weight=pos_weight)

    opt = torch.optim.AdamW(params, lr=lr, weight_decay=weight_decay)
    gen = torch.Generator().manual_seed(seed)
    hist = []
    n = len(y)
    for ep in range(epochs):
        perm = torch.randperm(n, generator=gen)
        for s in range(0, n, batch):
            idx = perm[s:s + batch]
            opt.zero_grad()
            loss = loss_fn(forward(xz[idx]), yt[idx])
            loss.backward()
            opt.step()
        with torch.no_grad():
            z = forward(xz)
            hist.append(dict(epoch=ep, loss=float(loss_fn(z, yt)), auc=auc(z.numpy(), y)))
    out = [p.detach().numpy().astype(np.float32) for p in params]
    mu32, sd32 = mu.astype(np.float32), sd.astype(np.float32)
    if kind == "mlp3":
        gate = {"w1": out[0], "b1": out[1], "w2": out[2][0], "b2": out[3], "mu": mu32, "sd": sd32}
    else:
        gate = {"kind": kind, "W": out[0::2], "b": out[1::2], "mu": mu32, "sd": sd32}
    return gate, hist


def load_trained_gate(ctx, gate):
    """Install a trained gate in a context (bag_load_gate)."""
    ctx.load_gate(synth.gate_flat(gate), gate["mu"], gate["sd"])
