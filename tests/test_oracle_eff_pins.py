"""Pins for the oracle's exploration efficiency Eff, Eq. (eq1): a hand-worked
branching graph, the paper's chain case (each trajectory one step) in closed form,
graph reachability by a library graph search, the ordering of the two readings and
their special cases.  CPU only."""
import json
import os

import numpy as np
import pytest

from paper_2606_18954_gb300 import workloads as W

HERE = os.path.dirname(os.path.abspath(__file__))
SMALL_TREE = W.TreeSpec("small-tree", 6, (2, 3, 3), 16, "f32", 6, 0.05, 0.9, ("per_step", 1, 9),
                        ("bernoulli", 0.5), p_stop=0.2)


def golden(name):
    with open(os.path.join(HERE, "golden", name)) as f:
        return json.load(f)


def test_eff_worked_example(oracle_mod):
    """Hand-derived Eff of the seven-state branching graph in both readings."""
    fx = golden("tree_micro.json")
    b = dict(group_rollout_off=np.asarray(fx["group_rollout_off"], np.int32),
             group_state_off=np.asarray(fx["group_state_off"], np.int32),
             group_token_off=np.asarray(fx["group_token_off"], np.int64),
             parent=np.asarray(fx["parent"], np.int32), step_len=np.asarray(fx["step_len"], np.int32),
             emb=np.asarray(fx["emb"], np.float32), emb_dtype="f32",
             reward=np.asarray(fx["reward"], np.uint8), layout="tree")
    out = oracle_mod.run(b, fx["params"], want=["eff_tree", "eff_graph"])
    assert out["eff_tree"][0] == pytest.approx(fx["eff_tree"], abs=1e-15)
    assert out["eff_graph"][0] == pytest.approx(fx["eff_graph"], abs=1e-15)


@pytest.mark.parametrize("name,groups", [("tiny", 8), ("agentic", 6), ("math", 3)])
def test_eff_chain_is_correct_trajectory_share(oracle_mod, name, groups):
    """Chain rollouts: each whole trajectory is one step, so Eff = tokens of the correct
    rollouts / all tokens (the paper's chain case), computed here from rewards and spans."""
    b = W.make_batch(W.CONFIGS[name].scaled(groups))
    out = oracle_mod.run(b, want=["eff_tree"])
    go, to, rw = b["group_rollout_off"], b["rollout_token_off"], b["reward"]
    for g in range(len(go) - 1):
        rr = np.arange(go[g], go[g + 1])
        L = (to[rr + 1] - to[rr]).astype(np.float64)
        assert out["eff_tree"][g] == pytest.approx((L * rw[rr]).sum() / L.sum(), rel=1e-14)


def _quotient_reach(b, labels):
    """States from which a correct leaf is reachable in the merged graph, by networkx
    reachability over the quotient digraph (class(p(v)) -> class(v))."""
    nx = pytest.importorskip("networkx")
    N = len(b["step_len"])
    tree = b.get("parent") is not None
    Gd = nx.DiGraph()
    Gd.add_nodes_from(set(labels.tolist()))
    targets = set()
    if tree:
        gs, go = b["group_state_off"], b["group_rollout_off"]
        for g in range(len(gs) - 1):
            s0, s1 = int(gs[g]), int(gs[g + 1])
            par = b["parent"][s0:s1]
            is_leaf = np.ones(s1 - s0, bool)
            is_leaf[par[par >= 0]] = False
            leaves = np.nonzero(is_leaf)[0]
            for k, v in enumerate(leaves):
                if b["reward"][go[g] + k]:
                    targets.add(int(labels[s0 + v]))
            for v in range(s1 - s0):
                if par[v] >= 0:
                    Gd.add_edge(int(labels[s0 + par[v]]), int(labels[s0 + v]))
    else:
        so = b["rollout_step_off"]
        for r in range(len(so) - 1):
            if b["reward"][r]:
                targets.add(int(labels[so[r + 1] - 1]))
            for v in range(so[r] + 1, so[r + 1]):
                Gd.add_edge(int(labels[v - 1]), int(labels[v]))
    good = set(targets)
    for t in targets:
        good |= nx.ancestors(Gd, t)
    return np.array([int(labels[v]) in good for v in range(N)])


@pytest.mark.parametrize("kind", ["chain", "tree"])
def test_eff_graph_by_library_reachability(oracle_mod, kind):
    b = W.make_batch(W.CONFIGS["tiny"].scaled(4)) if kind == "chain" else W.make_tree_batch(SMALL_TREE, seed=21)
    out = oracle_mod.run(b, want=["eff_graph", "class_id"])
    good = _quotient_reach(b, out["class_id"])
    sl = b["step_len"].astype(np.float64)
    N = len(sl)
    grp = np.empty(N, np.int64)
    if kind == "tree":
        gs = b["group_state_off"]
        for g in range(len(gs) - 1):
            grp[gs[g]:gs[g + 1]] = g
    else:
        go, so = b["group_rollout_off"], b["rollout_step_off"]
        for g in range(len(go) - 1):
            grp[so[go[g]]:so[go[g + 1]]] = g
    G = len(b["group_rollout_off"]) - 1
    want = np.bincount(grp, weights=sl * good, minlength=G) / np.bincount(grp, weights=sl, minlength=G)
    np.testing.assert_allclose(out["eff_graph"], want, rtol=1e-14)


@pytest.mark.parametrize("kind", ["chain", "tree"])
def test_eff_orderings_and_special_cases(oracle_mod, kind):
    b = W.make_batch(W.CONFIGS["tiny"].scaled(4)) if kind == "chain" else W.make_tree_batch(SMALL_TREE, seed=21)
    out = oracle_mod.run(b, want=["eff_tree", "eff_graph"])
    # merging only adds routes to a correct answer
    assert (out["eff_graph"] >= out["eff_tree"] - 1e-15).all()
    assert ((out["eff_tree"] >= 0) & (out["eff_graph"] <= 1)).all()
    # no merges: both readings coincide
    none = oracle_mod.run(b, dict(kappa=2.0), want=["eff_tree", "eff_graph"])
    np.testing.assert_array_equal(none["eff_tree"], none["eff_graph"])
    np.testing.assert_array_equal(none["eff_tree"], out["eff_tree"])  # the tree reading ignores merges
    # all rollouts correct: every step is; none correct: no step is
    for val in (1, 0):
        bb = dict(b, reward=np.full_like(b["reward"], val))
        o = oracle_mod.run(bb, want=["eff_tree", "eff_graph"])
        np.testing.assert_array_equal(o["eff_tree"], float(val))
        np.testing.assert_array_equal(o["eff_graph"], float(val))
