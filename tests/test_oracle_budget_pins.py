"""Pins for the oracle's per-layer merge and next-layer budgets (Sec. 4.2 budget halving,
Algorithm S.1 Stage 1): hand-worked budgets layer by layer, the classes of every layer
against library connected components of the explicit non-causal links, redundancy as
"not the first member of its class in registration order", conservation of the budget,
and the no-merge case.  CPU only."""
import json
import os

import numpy as np
import pytest

from oracle import budget as OB
from paper_2606_18954_gb300 import workloads as W

HERE = os.path.dirname(os.path.abspath(__file__))
SMALL = W.TreeSpec("small-tree", 5, (3, 3, 2, 2), 16, "f32", 5, 0.05, 0.9, ("per_step", 1, 9),
                   ("bernoulli", 0.5), p_stop=0.2)


def golden(name):
    with open(os.path.join(HERE, "golden", name)) as f:
        return json.load(f)


def micro_batch():
    fx = golden("tree_micro.json")
    b = dict(group_rollout_off=np.asarray(fx["group_rollout_off"], np.int32),
             group_state_off=np.asarray(fx["group_state_off"], np.int32),
             group_token_off=np.asarray(fx["group_token_off"], np.int64),
             parent=np.asarray(fx["parent"], np.int32), step_len=np.asarray(fx["step_len"], np.int32),
             emb=np.asarray(fx["emb"], np.float32), emb_dtype="f32",
             reward=np.asarray(fx["reward"], np.uint8), layout="tree")
    return b, fx["params"]


def test_budget_worked_example(oracle_mod):
    b, params = micro_batch()
    for case in golden("budget_micro.json")["cases"]:
        t = W.truncate_tree(b, case["layer"])
        full = np.ones(len(b["parent"]), np.uint8)
        for v in case.get("active_off", []):
            full[v] = 0
        act = full[t["source_states"]]
        got = OB.layer_budget(t, case["layer"], case["b_next"], act, params)["budget"]
        want = np.zeros(len(b["parent"]), np.int64)
        want[t["source_states"]] = got
        np.testing.assert_array_equal(want, case["budget"], err_msg=str(case))


def _components(t, kappa):
    """Min-index class labels of the explicit non-causal links (scipy components)."""
    from scipy.sparse import coo_matrix
    from scipy.sparse.csgraph import connected_components
    Z = t["emb"].astype(np.float64)
    N = len(Z)
    rows, cols = [], []
    gs = t["group_state_off"]
    for g in range(len(gs) - 1):
        s0, s1 = int(gs[g]), int(gs[g + 1])
        end = W.subtree_end(t["parent"][s0:s1])
        for i in range(s1 - s0):
            for j in range(i + 1, s1 - s0):
                if j < end[i]:
                    continue  # j lies in i's subtree (pre-order): ancestor-related
                zi, zj = Z[s0 + i], Z[s0 + j]
                den = np.linalg.norm(zi) * np.linalg.norm(zj)
                if den > 0 and zi @ zj / den >= kappa:
                    rows.append(s0 + i)
                    cols.append(s0 + j)
    A = coo_matrix((np.ones(len(rows)), (rows, cols)), shape=(N, N))
    _, comp = connected_components(A, directed=False)
    lab = np.empty(N, np.int64)
    for c in np.unique(comp):
        m = np.nonzero(comp == c)[0]
        lab[m] = m.min()
    return lab


@pytest.mark.parametrize("seed", [3, 4])
def test_layer_classes_are_components_and_final_layer_is_the_batch(oracle_mod, seed):
    b = W.make_tree_batch(SMALL, seed=seed)
    H = len(SMALL.schedule)
    for h in range(1, H + 1):
        t = W.truncate_tree(b, h)
        got = OB.layer_budget(t, h, 2, t["active"], dict(kappa=SMALL.kappa))["class_id"]
        np.testing.assert_array_equal(got, _components(t, SMALL.kappa), err_msg=f"layer {h}")
    # after the last layer the per-layer merge has compared every non-causal pair once:
    # the classes of the whole batch
    whole = oracle_mod.run(b, dict(kappa=SMALL.kappa), want=["class_id"])["class_id"]
    np.testing.assert_array_equal(OB.layer_budget(W.truncate_tree(b, H), H, 2, None,
                                                  dict(kappa=SMALL.kappa))["class_id"], whole)


@pytest.mark.parametrize("b_next", [1, 2, 3, 5])
def test_redundancy_is_not_first_in_registration_order_and_budget_is_conserved(oracle_mod, b_next):
    b = W.make_tree_batch(SMALL.scaled(8), seed=7)
    for h in range(1, len(SMALL.schedule) + 1):
        t = W.truncate_tree(b, h)
        res = OB.layer_budget(t, h, b_next, t["active"], dict(kappa=SMALL.kappa))
        dep = W.tree_depths(t)
        lab = res["class_id"]
        gs = t["group_state_off"]
        for g in range(len(gs) - 1):
            s0, s1 = int(gs[g]), int(gs[g + 1])
            v = np.arange(s0, s1)
            order = v[np.lexsort((v, dep[v]))]  # registration order: layer, then index
            _, first = np.unique(lab[order], return_index=True)
            firsts = set(order[first].tolist())
            fr = v[res["frontier"][v]]
            for x in fr:
                assert res["redundant"][x] == (x not in firsts)
            k = sum(1 for x in fr if x in firsts)
            total = int(res["budget"][v].sum())
            if k > 0:
                assert total == b_next * len(fr)  # the saved budget is spent in full
            else:
                assert total == max(1, b_next // 2) * len(fr)
            assert (res["budget"][fr] >= 1).all()
            assert (res["budget"][v[~res["frontier"][v]]] == 0).all()


def test_no_merges_gives_the_schedule(oracle_mod):
    b = W.make_tree_batch(SMALL, seed=5)
    for h in range(1, len(SMALL.schedule) + 1):
        t = W.truncate_tree(b, h)
        res = OB.layer_budget(t, h, 3, t["active"], dict(kappa=2.0))
        np.testing.assert_array_equal(res["budget"], 3 * res["frontier"].astype(np.int64))
