"""Mutation checks of the policy-loss and per-layer-budget oracles (CPU only): each test
plants one plausible mistake in the oracle (a dropped factor, a swapped operand, a wrong
rule) and asserts that at least one of the oracle's pins then fails.  Pins that no mutant
can get past are what makes the oracle trustworthy without an implementation to compare
against."""
import numpy as np
import pytest

import test_oracle_budget_pins as BP
import test_oracle_loss_pins as LP
from oracle import budget as OB
from oracle import loss as OL


def _fails(pins):
    """True when at least one of the pins (zero-argument callables) fails."""
    for pin in pins:
        try:
            pin()
        except AssertionError:
            return True
    return False


# ---------------------------------------------------------------- loss oracle mutants

def _weights_without_edge_length(batch, norm="edge"):
    edge, _ = OL.edge_of_token(batch)
    grp = OL.group_of_state(batch)
    G = len(batch["group_rollout_off"]) - 1
    n_edges = np.bincount(grp, minlength=G).astype(np.float64)
    if norm == "token":
        return np.full(len(edge), 1.0 / len(edge))
    return 1.0 / (float(np.count_nonzero(n_edges)) * n_edges[grp[edge]])  # 1/|e| dropped


def _weights_over_all_groups(batch, norm="edge"):
    edge, elen = OL.edge_of_token(batch)
    if norm == "token":
        return np.full(len(edge), 1.0 / len(edge))
    grp = OL.group_of_state(batch)
    G = len(batch["group_rollout_off"]) - 1
    n_edges = np.bincount(grp, minlength=G).astype(np.float64)
    return 1.0 / (G * n_edges[grp[edge]] * elen)  # empty groups counted in G'


def _surrogate_max(ratio, A, lo, hi):
    u, c = ratio * A, np.clip(ratio, 1 - lo, 1 + hi) * A
    take = u >= c
    return np.maximum(u, c), np.where(take, ratio * A, 0.0), ~take


def _surrogate_grad_always(ratio, A, lo, hi):
    u, c = ratio * A, np.clip(ratio, 1 - lo, 1 + hi) * A
    return np.minimum(u, c), ratio * A, ~(u <= c)  # gradient also through the clipped branch


def _surrogate_clip_grad(ratio, A, lo, hi):
    u, c = ratio * A, np.clip(ratio, 1 - lo, 1 + hi) * A
    take = u <= c
    return np.minimum(u, c), np.where(take, c, 0.0), ~take  # derivative of clip(r) A


def _surrogate_bounds_swapped(ratio, A, lo, hi):
    u, c = ratio * A, np.clip(ratio, 1 - hi, 1 + lo) * A
    take = u <= c
    return np.minimum(u, c), np.where(take, ratio * A, 0.0), ~take


def _weights_token_norm_per_edge(batch, norm="edge"):
    edge, elen = OL.edge_of_token(batch)
    if norm == "token":
        return 1.0 / (len(np.unique(edge)) * elen)  # "token" taken as a mean over edges
    grp = OL.group_of_state(batch)
    G = len(batch["group_rollout_off"]) - 1
    n_edges = np.bincount(grp, minlength=G).astype(np.float64)
    return 1.0 / (float(np.count_nonzero(n_edges)) * n_edges[grp[edge]] * elen)


def _kl_wrong_sign(x):
    return np.expm1(x) + x, -np.expm1(x)


def _kl_wrong_derivative(x):
    return np.expm1(x) - x, np.expm1(x)


LOSS_MUTANTS = {
    "no 1/|e|": ("token_weights", _weights_without_edge_length),
    "G' counts empty groups": ("token_weights", _weights_over_all_groups),
    "max instead of min": ("surrogate", _surrogate_max),
    "gradient through clipped branch": ("surrogate", _surrogate_grad_always),
    "derivative of the clipped term": ("surrogate", _surrogate_clip_grad),
    "clip bounds swapped": ("surrogate", _surrogate_bounds_swapped),
    "token normalisation as an edge mean": ("token_weights", _weights_token_norm_per_edge),
    "k3 sign": ("kl_k3", _kl_wrong_sign),
    "k3 derivative sign": ("kl_k3", _kl_wrong_derivative),
}


def _loss_pins(oracle_mod):
    return [
        LP.test_loss_worked_example_dual,
        LP.test_loss_worked_example_decoupled_clip,
        LP.test_loss_worked_example_kl,
        LP.test_loss_worked_example_split,
        lambda: LP.test_loss_at_ratio_one(oracle_mod, "chain"),
        lambda: LP.test_loss_gradient_matches_finite_differences(oracle_mod, "chain", "dual", "edge", 0.05),
    ]


@pytest.mark.parametrize("name", sorted(LOSS_MUTANTS))
def test_loss_pins_catch_mutant(oracle_mod, monkeypatch, name):
    attr, fn = LOSS_MUTANTS[name]
    monkeypatch.setattr(OL, attr, fn)
    assert _fails(_loss_pins(oracle_mod)), f"no pin catches the mutant: {name}"


def test_loss_pins_catch_split_mask_ignored(oracle_mod, monkeypatch):
    orig = OL.token_loss

    def mutant(batch, logp, old_logp, ref_logp=None, edge_mask=None, **kw):
        ones = None if edge_mask is None else np.ones_like(np.asarray(edge_mask))
        return orig(batch, logp, old_logp, ref_logp, edge_mask=ones, **kw)

    monkeypatch.setattr(OL, "token_loss", mutant)
    assert _fails(_loss_pins(oracle_mod))


def test_unmutated_loss_oracle_passes(oracle_mod):
    assert not _fails(_loss_pins(oracle_mod))


# -------------------------------------------------------------- budget oracle mutants

BUDGET_MUTANTS = {
    "halving without the floor of one": ("halved", lambda b: b // 2),
    "no halving": ("halved", lambda b: b),
    "registration by index only": ("registered_before", lambda dep, u, v: u < v),
    "registration by layer only": ("registered_before", lambda dep, u, v: dep[u] < dep[v]),
    "registration in reverse index order": ("registered_before",
                                            lambda dep, u, v: dep[u] < dep[v] or (dep[u] == dep[v] and u > v)),
    "registration with later layers first": ("registered_before",
                                             lambda dep, u, v: dep[u] > dep[v] or (dep[u] == dep[v] and u < v)),
    "remainder to the last states": ("spread", lambda saved, k: [saved // k + (1 if r >= k - saved % k else 0)
                                                                for r in range(k)]),
    "savings not spent": ("spread", lambda saved, k: [0] * k),
}


def _budget_pins(oracle_mod):
    return [
        lambda: BP.test_budget_worked_example(oracle_mod),
        lambda: BP.test_redundancy_is_not_first_in_registration_order_and_budget_is_conserved(oracle_mod, 3),
        lambda: BP.test_no_merges_gives_the_schedule(oracle_mod),
    ]


@pytest.mark.parametrize("name", sorted(BUDGET_MUTANTS))
def test_budget_pins_catch_mutant(oracle_mod, monkeypatch, name):
    attr, fn = BUDGET_MUTANTS[name]
    monkeypatch.setattr(OB, attr, fn)
    assert _fails(_budget_pins(oracle_mod)), f"no pin catches the mutant: {name}"


def test_budget_pins_catch_inactive_states_on_the_frontier(oracle_mod, monkeypatch):
    orig = OB.layer_budget

    def mutant(batch, layer, b_next, active=None, params=None):
        return orig(batch, layer, b_next, None, params)  # every state of the layer expanded

    monkeypatch.setattr(OB, "layer_budget", mutant)
    assert _fails(_budget_pins(oracle_mod))


def test_unmutated_budget_oracle_passes(oracle_mod):
    assert not _fails(_budget_pins(oracle_mod))
