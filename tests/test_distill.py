"""Host logic of the offline side (Algorithm 1 at toy scale): the matched-NFE reference
search of Eq. 2 against the oracle's brute-force argmin, and the gate distillation of
Eq. 4 against the oracle's loss definition.  No GPU: the distances here are synthetic
functions or oracle rollouts."""

import itertools

import numpy as np
import pytest

from oracle import bag_oracle as O
from paper_2608_09231_gb300 import configs, distill, synth


def test_mask_starts_and_moves():
    for T, B in [(10, 4), (7, 7), (9, 1), (50, 13)]:
        for m in (distill.uniform_mask(B, T), distill.front_loaded_mask(B, T)):
            assert len(m) == T and sum(m) == B and m[0] == 1
        nb = distill.neighbors(distill.uniform_mask(B, T))
        assert len(nb) == (B - 1) * (T - B)
        assert len({tuple(m) for m in nb}) == len(nb)
        assert all(sum(m) == B and m[0] == 1 for m in nb)
    assert distill.uniform_mask(4, 10) == O.static_uniform_schedule(4, 10)
    lo = distill.uniform_mask(3, 12)
    hi = distill.insert_steps(lo, 6)
    assert sum(hi) == 6 and all(h >= l for h, l in zip(hi, lo))
    hi2 = distill.insert_steps(lo, 6, rng=np.random.default_rng(1))
    assert sum(hi2) == 6 and all(h >= l for h, l in zip(hi2, lo))


def test_oracle_enumeration_covers_every_matched_nfe_mask():
    masks = list(O.all_masks(4, 9))
    assert len(masks) == 56   # C(8, 3)
    assert all(m[0] == 1 and sum(m) == 4 for m in masks)
    w = np.arange(9.0)[::-1]
    m, dv = O.reference_by_enumeration(lambda m: float(np.dot(m, w)), 4, 9)
    assert m == [1, 0, 0, 0, 0, 0, 1, 1, 1] and dv == w[0] + w[6] + w[7] + w[8]


def test_search_finds_the_optimum_of_additive_distances():
    """With an additive distance every swap-local optimum is global: the search must land
    on Eq. 2's argmin from any start."""
    rng = np.random.default_rng(0)
    for T, B in [(10, 4), (16, 7), (12, 2)]:
        w = rng.normal(size=T)
        dist = lambda m: float(np.dot(m, w))  # noqa: E731
        want, dw = O.reference_by_enumeration(dist, B, T)
        got = distill.local_search(dist, B, T, [distill.uniform_mask(B, T)])
        assert got["mask"] == want and abs(got["distance"] - dw) < 1e-12


def test_search_with_annealing_on_interacting_distances():
    """Pairwise interactions make the landscape rugged; the annealed multi-start search
    reaches the brute-force optimum on these seeded instances and never returns worse
    than its best start."""
    T, B = 9, 4
    hits = 0
    for seed in range(6):
        rng = np.random.default_rng(seed)
        w, J = rng.normal(size=T), rng.normal(size=(T, T))

        def dist(m):
            m = np.asarray(m, float)
            return float(m @ w + m @ np.triu(J, 1) @ m)

        want, dw = O.reference_by_enumeration(dist, B, T)
        starts = [distill.uniform_mask(B, T), distill.front_loaded_mask(B, T)]
        got = distill.local_search(dist, B, T, starts, rng=np.random.default_rng(seed),
                                   anneal_steps=30)
        assert got["distance"] <= min(dist(s) for s in starts) + 1e-12
        assert got["evals"] <= 56
        hits += abs(got["distance"] - dw) < 1e-12
    assert hits >= 5


def test_search_on_oracle_rollouts_matches_enumeration():
    """Eq. 2 on a real (oracle) model: D = mean squared error of x_T(m) to the uncached
    output, T = 6, B = 3 (ten masks)."""
    cfg = configs.get_config("tiny_ragged")
    W, g, inp = synth.make_weights(cfg), synth.make_gate(cfg["gate_seed"]), synth.make_inputs(cfg)
    T, B = 6, 3
    target = O.sample(cfg, W, g, inp, T=T, B=T, policy="full")["x"]
    cache = {}

    def dist(m):
        k = tuple(m)
        if k not in cache:
            cache[k] = float(np.mean((O.sample(cfg, W, g, inp, T=T, B=B, policy=list(m))["x"]
                                      - target) ** 2))
        return cache[k]

    want, dw = O.reference_by_enumeration(dist, B, T)
    got = distill.local_search(dist, B, T, [distill.uniform_mask(B, T),
                                            distill.front_loaded_mask(B, T)],
                               anneal_steps=10)
    assert got["mask"] == want and got["distance"] == dw


def _examples(n=400, seed=0, kind="flux6"):
    rng = np.random.default_rng(seed)
    k = 3 if kind == "mlp3" else 6
    X = rng.normal(size=(n, k)) * [0.3, 2.0, 0.5, 4.0, 0.1, 0.05][:k] + [0.4, 1.0, 0.0, 2.0, 0.2, 0.1][:k]
    # separable labels with a margin, 1 positive in 4 (class imbalance)
    s = (X[:, 1] - 1.0) / 2.0 + (X[:, k - 1] - X[:, k - 1].mean()) / X[:, k - 1].std()
    thr = np.quantile(s, 0.75)
    keep = np.abs(s - thr) > 0.15
    return X[keep], (s[keep] > thr).astype(float)


@pytest.mark.parametrize("kind", ["flux6", "wan6", "mlp3"])
def test_fit_gate_loss_is_eq4_and_separates(kind):
    X, y = _examples(kind=kind)
    gate, hist = distill.fit_gate(X, y, kind=kind, epochs=300, lr=3e-3, weight_decay=1e-4)
    mu, sd = O.zscore_stats(X)
    assert np.allclose(gate["mu"], mu, rtol=1e-6) and np.allclose(gate["sd"], sd, rtol=1e-6)
    # the trainer's objective is the oracle's Eq. 4 (class-balanced, z-scored)
    ref = O.distillation_loss(gate, X, y)
    assert abs(hist[-1]["loss"] - ref) <= 1e-4 * max(1.0, ref)
    assert hist[-1]["loss"] < 0.5 * hist[0]["loss"]
    z = O.gate_forward64(gate, (X - gate["mu"]) / gate["sd"])
    assert distill.auc(z, y) > 0.99
    assert np.mean((z > 0) == (y > 0.5)) > 0.97


def test_fit_gate_weights_the_positive_class():
    """Class balancing: on overlapping classes at 1:9, the weighted loss puts the decision
    where both classes count equally, so the gate calls far more than 10 % positive."""
    rng = np.random.default_rng(3)
    n = 2000
    y = (rng.random(n) < 0.1).astype(float)
    X = rng.normal(size=(n, 6)) + y[:, None] * 0.8
    gate, _ = distill.fit_gate(X, y, kind="flux6", epochs=100, lr=3e-3)
    z = O.gate_forward64(gate, (X - gate["mu"]) / gate["sd"])
    assert np.mean(z > 0) > 0.25


def test_trained_gate_in_the_decision_path():
    """The exported gate (seeded-generator layout, loadable by bag_load_gate) evaluates in
    the fixed-order fp32 decision path to the float64 logit up to fp32 rounding."""
    X, y = _examples(n=200, seed=5)
    gate, _ = distill.fit_gate(X, y, kind="flux6", epochs=50)
    flat = synth.gate_flat(gate)
    assert flat.size == 449
    z64 = O.gate_forward64(gate, (X - gate["mu"]) / gate["sd"])
    for i in range(0, len(X), 17):
        z32 = O.gate_logit6([np.float32(v) for v in X[i]], gate)
        assert abs(float(z32) - z64[i]) <= 1e-4 * max(1.0, abs(z64[i]))


def test_auc_definition():
    y = np.array([0, 0, 1, 1, 0, 1])
    s = np.array([0.1, 0.4, 0.35, 0.8, 0.4, 0.4])
    pairs = [(p, n) for p, n in itertools.product(s[y == 1], s[y == 0])]
    want = np.mean([1.0 if p > n else 0.5 if p == n else 0.0 for p, n in pairs])
    assert abs(distill.auc(s, y) - want) < 1e-12
