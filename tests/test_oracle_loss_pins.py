"""Pins for the oracle's GraphPO policy loss (Sec. 4.5 objective, Algorithm S.1
Stage 4): a hand-worked five-token example in every form, the gradient against
central finite differences of the loss, closed forms at ratio 1, the split form's
reduction to the dual form where nothing is clipped, and the KL estimate's special
values.  CPU only."""
import json
import math
import os

import numpy as np
import pytest

from oracle import loss as OL
from paper_2606_18954_gb300 import workloads as W

HERE = os.path.dirname(os.path.abspath(__file__))


def golden(name):
    with open(os.path.join(HERE, "golden", name)) as f:
        return json.load(f)


def _micro():
    fx = golden("loss_micro.json")
    b = {k: np.asarray(v) for k, v in fx["batch"].items()}
    b["step_len"] = b["step_len"].astype(np.int32)
    old = np.full(len(fx["ratio"]), fx["old_logp"])
    logp = old + np.log(np.asarray(fx["ratio"]))
    return fx, b, logp, old


def test_loss_worked_example_dual():
    fx, b, logp, old = _micro()
    d = fx["dual"]
    out = OL.token_loss(b, logp, old, edge_adv=d["edge_adv"])
    assert out["loss"] == pytest.approx(d["loss"], abs=1e-15)
    np.testing.assert_allclose(out["grad"], d["grad"], rtol=1e-14, atol=1e-16)
    assert out["clipped"] == d["clipped"]
    assert out["ratio_mean"] == pytest.approx(d["ratio_mean"], abs=1e-15)
    t = fx["dual_token_norm"]
    out = OL.token_loss(b, logp, old, edge_adv=d["edge_adv"], norm="token")
    assert out["loss"] == pytest.approx(t["loss"], abs=1e-15)
    np.testing.assert_allclose(out["grad"], t["grad"], rtol=1e-14, atol=1e-16)


def test_loss_worked_example_decoupled_clip():
    fx, b, logp, old = _micro()
    c = fx["dual_decoupled_clip"]
    out = OL.token_loss(b, logp, old, edge_adv=fx["dual"]["edge_adv"], clip_low=c["clip_low"],
                        clip_high=c["clip_high"])
    assert out["loss"] == pytest.approx(c["loss"], abs=1e-15)
    np.testing.assert_allclose(out["grad"], c["grad"], rtol=1e-14, atol=1e-16)
    assert out["clipped"] == c["clipped"]


def test_loss_worked_example_kl():
    fx, b, logp, old = _micro()
    k = fx["dual_kl"]
    ref = logp + np.asarray(fx["kl_x"])
    out = OL.token_loss(b, logp, old, ref, edge_adv=fx["dual"]["edge_adv"], beta=k["beta"])
    assert out["kl"] == pytest.approx(k["kl"], abs=1e-15)
    assert out["loss"] == pytest.approx(k["loss"], abs=1e-15)
    np.testing.assert_allclose(out["grad"], k["grad"], rtol=1e-14, atol=1e-16)


def test_loss_worked_example_split():
    fx, b, logp, old = _micro()
    s = fx["split"]
    out = OL.token_loss(b, logp, old, edge_cor=s["edge_cor"], edge_eff=s["edge_eff"], edge_mask=s["edge_mask"],
                        lambda_eff=s["lambda_eff"], form="split")
    assert out["loss"] == pytest.approx(s["loss"], abs=1e-15)
    np.testing.assert_allclose(out["grad"], s["grad"], rtol=1e-14, atol=1e-16)
    assert out["clipped"] == s["clipped"]


SMALL_CHAIN = W.Spec("small-chain", 3, 4, 16, "f32", 4, 0.05, 0.9, ("uniform", 2, 5), ("per_step", 1, 6),
                     ("bernoulli", 0.5))


def _case(oracle_mod, kind, seed):
    if kind == "chain":
        b = W.make_batch(SMALL_CHAIN, seed=seed)
    else:
        spec = W.TreeSpec("small-tree", 3, (2, 3, 2), 16, "f32", 6, 0.05, 0.9, ("per_step", 1, 6),
                          ("bernoulli", 0.5), p_stop=0.2)
        b = W.make_tree_batch(spec, seed=seed)
    adv = oracle_mod.run(b, want=["edge_adv", "a_cor", "e_eff", "edge_eff_mask"])
    T = int(b["group_token_off"][-1] if kind == "tree" else b["rollout_token_off"][-1])
    lp = W.make_logprobs(T, seed + 1)
    return b, adv, lp


@pytest.mark.parametrize("kind", ["chain", "tree"])
@pytest.mark.parametrize("form,norm,beta", [("dual", "edge", 0.0), ("dual", "token", 0.05), ("split", "edge", 0.1),
                                            ("split", "token", 0.0)])
def test_loss_gradient_matches_finite_differences(oracle_mod, kind, form, norm, beta):
    """dL/dlogp of every token against central differences of the oracle's own loss
    (the margin keeps every ratio 1e-4 from a clip bound, far beyond the step)."""
    b, adv, lp = _case(oracle_mod, kind, 31)
    kw = dict(edge_adv=adv["edge_adv"], edge_cor=adv["a_cor"], edge_eff=adv["e_eff"], edge_mask=adv["edge_eff_mask"],
              form=form, norm=norm, beta=beta, lambda_eff=0.7)
    logp = lp["logp"].astype(np.float64)
    base = OL.token_loss(b, logp, lp["old_logp"], lp["ref_logp"], **kw)
    rng = np.random.default_rng(5)
    idx = rng.choice(len(logp), size=min(40, len(logp)), replace=False)
    h = 1e-5  # ratios stay >= 8e-5 (in log) from a clip bound
    for t in idx:
        up, dn = logp.copy(), logp.copy()
        up[t] += h
        dn[t] -= h
        fd = (OL.token_loss(b, up, lp["old_logp"], lp["ref_logp"], **kw)["loss"]
              - OL.token_loss(b, dn, lp["old_logp"], lp["ref_logp"], **kw)["loss"]) / (2 * h)
        assert fd == pytest.approx(base["grad"][t], rel=1e-5, abs=1e-9 * abs(base["weights"][t]) + 1e-13)


@pytest.mark.parametrize("kind", ["chain", "tree"])
def test_loss_at_ratio_one(oracle_mod, kind):
    """logp = old_logp: every ratio is 1, nothing is clipped, and J is the mean over the
    groups of the mean over their edges of A (edge normalisation), or the token-weighted
    mean of A (token normalisation); the gradient is -w A."""
    b, adv, lp = _case(oracle_mod, kind, 41)
    old = lp["old_logp"].astype(np.float64)
    A = adv["edge_adv"]
    grp = OL.group_of_state(b)
    G = len(b["group_rollout_off"]) - 1
    per_group = [A[grp == g].mean() for g in range(G) if (grp == g).any()]
    out = OL.token_loss(b, old, old, edge_adv=A)
    assert out["clipped"] == 0 and out["ratio_mean"] == 1.0
    assert out["loss"] == pytest.approx(-np.mean(per_group), rel=1e-12, abs=1e-15)
    sl = b["step_len"].astype(np.float64)
    out = OL.token_loss(b, old, old, edge_adv=A, norm="token")
    assert out["loss"] == pytest.approx(-(sl * A).sum() / sl.sum(), rel=1e-12, abs=1e-15)


@pytest.mark.parametrize("kind", ["chain", "tree"])
def test_split_equals_dual_without_clipping(oracle_mod, kind):
    """With every ratio inside the clip range both surrogates are linear in A, so the split
    form with the oracle's A_cor, routed A_eff and m_eff equals the dual form on A_dual =
    A_cor + lambda A_eff (A_eff is 0 wherever m_eff is 0); lambda = 0 gives the dual
    form on A_cor at any ratio."""
    b, adv, lp = _case(oracle_mod, kind, 51)
    rng = np.random.default_rng(3)
    old = lp["old_logp"].astype(np.float64)
    logp = old + rng.uniform(-0.15, 0.15, len(old))  # ratios in [0.86, 1.17]
    lam = 0.6
    split = OL.token_loss(b, logp, old, edge_cor=adv["a_cor"], edge_eff=adv["e_eff"], edge_mask=adv["edge_eff_mask"],
                          lambda_eff=lam, form="split")
    dual = OL.token_loss(b, logp, old, edge_adv=adv["a_cor"] + lam * adv["e_eff"])
    assert split["loss"] == pytest.approx(dual["loss"], rel=1e-12, abs=1e-15)
    np.testing.assert_allclose(split["grad"], dual["grad"], rtol=1e-12, atol=1e-18)
    logp = lp["logp"].astype(np.float64)
    split = OL.token_loss(b, logp, old, edge_cor=adv["a_cor"], edge_eff=adv["e_eff"], edge_mask=adv["edge_eff_mask"],
                          lambda_eff=0.0, form="split")
    dual = OL.token_loss(b, logp, old, edge_adv=adv["a_cor"])
    assert split["loss"] == dual["loss"] and split["clipped"] == dual["clipped"]


def test_kl_estimate_special_values():
    """k3 = e^x - x - 1: zero when pi_ref = pi_theta, 1 - ln 2 at x = ln 2, x^2/2 to
    third order near 0, and never negative."""
    b = dict(group_rollout_off=np.array([0, 1]), rollout_step_off=np.array([0, 1]),
             rollout_token_off=np.array([0, 4]), step_len=np.array([4], np.int32), reward=np.array([1], np.uint8))
    logp = np.array([-1.0, -2.0, -0.5, -3.0])
    x = np.array([0.0, math.log(2.0), 1e-4, -5.0])
    out = OL.token_loss(b, logp, logp, logp + x, edge_adv=[0.0], beta=1.0)
    k = np.array([0.0, 1.0 - math.log(2.0), 1e-8 / 2 + 1e-12 / 6, math.exp(-5.0) + 4.0])
    assert out["kl"] == pytest.approx(k.mean(), rel=1e-12)
    assert out["loss"] == pytest.approx(k.mean(), rel=1e-12)  # A = 0: L = beta * KL
    np.testing.assert_allclose(out["grad"], -np.expm1(x) / 4, rtol=1e-12)  # beta w (1 - e^x)
