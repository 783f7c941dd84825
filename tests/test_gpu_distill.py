"""Algorithm 1 at toy scale on the GPU: rollouts under searched masks through the C ABI,
the reference search of Eq. 2 against the oracle's brute-force argmin, and a distilled
gate deployed by Algorithm 2 (bag_load_gate, bag_set_budget)."""

import numpy as np
import pytest
import torch

from oracle import bag_oracle as O
from paper_2608_09231_gb300 import bag, configs, distill, synth

pytestmark = pytest.mark.gpu


def test_rollout_distances_match_the_oracle(lib):
    cfg = configs.get_config("tiny_ragged")
    T = 8
    ctx = bag.create(cfg, T=T, B=3)
    inp = synth.make_inputs(cfg)
    ro = distill.Rollouts(ctx, inp)
    W, g = synth.make_weights(cfg), synth.make_gate(cfg["gate_seed"])
    target = O.sample(cfg, W, g, inp, T=T, B=T, policy="full")["x"]
    rms = float(np.sqrt(np.mean(target ** 2)))
    assert float(np.max(np.abs(ro.target() - target))) <= 1e-4 * rms
    rng = np.random.default_rng(0)
    for B in (2, 3, 5):
        for _ in range(2):
            m = [1] + list(rng.permutation([1] * (B - 1) + [0] * (T - B)))
            dg = ro.distance(m)
            do = float(np.mean((O.sample(cfg, W, g, inp, T=T, B=B, policy=m)["x"] - target) ** 2))
            # both are mean squares of latent differences; each latent within 1e-4 RMS
            assert abs(np.sqrt(dg) - np.sqrt(do)) <= 2e-4 * rms, (m, dg, do)
    ctx.close()


def test_search_with_gpu_rollouts_finds_the_oracle_optimum(lib):
    """Eq. 2 by the local search on GPU rollouts equals the brute-force argmin over the
    oracle's rollouts (T = 8, B = 3: 21 masks), up to distances the two cannot separate."""
    cfg = configs.get_config("tiny_ragged")
    T, B = 8, 3
    ctx = bag.create(cfg, T=T, B=B)
    inp = synth.make_inputs(cfg, sample_seed=2)
    ro = distill.Rollouts(ctx, inp)
    got = distill.local_search(ro.distance, B, T, [distill.uniform_mask(B, T),
                                                   distill.front_loaded_mask(B, T)],
                               anneal_steps=10)
    ctx.close()
    W, g = synth.make_weights(cfg), synth.make_gate(cfg["gate_seed"])
    target = O.sample(cfg, W, g, inp, T=T, B=T, policy="full")["x"]
    rms = float(np.sqrt(np.mean(target ** 2)))

    def dist(m):
        return float(np.mean((O.sample(cfg, W, g, inp, T=T, B=B, policy=list(m))["x"] - target) ** 2))

    want, dw = O.reference_by_enumeration(dist, B, T)
    d_got = dist(got["mask"])
    assert np.sqrt(d_got) - np.sqrt(dw) <= 4e-4 * rms, (got["mask"], want, d_got, dw)


def test_algorithm1_distilled_gate_deploys_budget_exact(lib):
    """Search references for three inputs at three budgets, fit the paper's FLUX gate
    (6-8-8-32-1) on the logged states, load it, and sample held-out inputs at a budget it
    was not trained on: NFE = B, and every logged logit is the oracle's fp32 logit of the
    trained gate on the logged inputs (bit for bit)."""
    cfg = configs.get_config("tiny_ragged", gate_kind="flux6")
    T = 10
    ctx = bag.create(cfg, T=T, B=4)
    inputs = [synth.make_inputs(cfg, sample_seed=s) for s in range(3)]
    X, y, cells = distill.reference_examples(ctx, inputs, budgets=(3, 5, 7), kind="flux6",
                                             anneal_steps=8, max_evals=80)
    assert X.shape == (9 * (T - 1), 6) and set(np.unique(y)) <= {0.0, 1.0}
    for c in cells:
        assert sum(c["mask"]) == c["B"] and c["mask"][0] == 1
        u = distill.uniform_mask(c["B"], T)
        assert c["distance"] <= distill.Rollouts(ctx, inputs[c["input"]]).distance(u) + 1e-12
    gate, hist = distill.fit_gate(X, y, kind="flux6", epochs=300, lr=1e-3, weight_decay=1e-4)
    assert hist[-1]["loss"] < hist[0]["loss"]
    distill.load_trained_gate(ctx, gate)
    ctx.set_policy(bag.POLICY_BAG)
    B = 4
    ctx.set_budget(B)
    for s in (10, 11):
        inp = synth.make_inputs(cfg, sample_seed=s)
        x = torch.from_numpy(inp["x"].copy()).cuda()
        ctx.reset()
        m, log, nfe = ctx.run(x, torch.from_numpy(inp["txt"]).cuda(),
                              torch.from_numpy(inp["pooled"]).cuda())
        torch.cuda.synchronize()
        assert nfe == B and int(m.sum()) == B and m[0] == 1
        bits = [None]
        for t in range(1, T):
            f = [np.float32(v) for v in log[t, distill.LOG_COLS["flux6"]]]
            z = O.gate_logit6(f, gate)
            assert z == np.float32(log[t, 3]), t
            bits.append(1 if z > O.gate_threshold(0.5) else 0)
        assert list(m) == O.schedule_from_gate_bits(bits, B, T)
    ctx.close()
