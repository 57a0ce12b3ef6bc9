"""Pins for the CPU oracle: each check fixes the oracle to something other than
itself -- a hand-worked example, a closed form, a textbook or library routine,
an invariant the paper states, brute force on tiny inputs, or the generator's
planted ground truth.  CPU only."""
import json
import math
import os

import numpy as np
import pytest
from scipy.sparse import csr_matrix
from scipy.sparse.csgraph import connected_components

from batches import emb_f64, from_rollouts, states_of
from paper_2606_18954_gb300 import workloads as W

HERE = os.path.dirname(os.path.abspath(__file__))
E = np.eye(8)


def golden(name):
    with open(os.path.join(HERE, "golden", name)) as f:
        return json.load(f)


# ------------------------------------------------------------------ worked example


def _micro_batch(fx, root_emb=None):
    b = dict(group_rollout_off=np.asarray(fx["group_rollout_off"], np.int32),
             rollout_step_off=np.asarray(fx["rollout_step_off"], np.int32),
             step_len=np.asarray(fx["step_len"], np.int32),
             emb=np.asarray(fx["emb"], np.float32), emb_dtype="f32",
             reward=np.asarray(fx["reward"], np.uint8))
    so, sl = b["rollout_step_off"], b["step_len"]
    to = np.zeros(len(so), np.int64)
    for r in range(len(so) - 1):
        to[r + 1] = to[r] + sl[so[r]:so[r + 1]].sum()
    b["rollout_token_off"] = to
    if root_emb is not None:
        b["root_emb"] = np.asarray(root_emb, np.float32)
    return b


def test_micro_worked_example(oracle_mod):
    """Hand-derived values of a 3-rollout x 2-step graph (Sec. 4.2-4.5)."""
    fx = golden("micro_3x2.json")
    out = oracle_mod.run(_micro_batch(fx), fx["params"])
    for key, val in fx["expected"].items():
        got = out[key]
        if key in ("class_id", "cor_group_size", "edge_eff_mask"):
            np.testing.assert_array_equal(got, np.asarray(val), err_msg=key)
        else:
            np.testing.assert_allclose(got, np.asarray(val), rtol=1e-12, atol=1e-15, err_msg=key)
    # every token of an edge carries the edge's A_dual (Sec. 4.5)
    want = np.repeat(np.asarray(fx["expected"]["edge_adv"]), fx["step_len"])
    np.testing.assert_allclose(out["adv"], want, rtol=1e-12, atol=1e-15)
    np.testing.assert_array_equal(out["eff_mask"], np.repeat(fx["expected"]["edge_eff_mask"], fx["step_len"]))


def test_micro_root_embedding_variant(oracle_mod):
    """With a root embedding, eta on root edges uses it (Sec. 4.3 r_step on (v0, v))."""
    fx = golden("micro_3x2.json")
    out = oracle_mod.run(_micro_batch(fx, fx["root_emb_variant"]["root_emb"]), fx["params"])
    exp = fx["root_emb_variant"]["a_cor_root_edges"]
    np.testing.assert_allclose(out["a_cor"][[0, 2, 4]], [exp["A1"], exp["B1"], exp["C1"]], rtol=1e-12)
    np.testing.assert_allclose(out["eta"][[0, 2, 4]], [1.0, 1.0, 0.0], atol=1e-15)


# ------------------------------------------------------------------ classes


def _components(batch, kappa, same_depth=False):
    """Connected components of the thresholded comparable-pair graph, via scipy."""
    roll, depth, grp = states_of(batch)
    Z = emb_f64(batch)
    nrm = np.linalg.norm(Z, axis=1)
    Zn = Z / np.where(nrm == 0, 1, nrm)[:, None]
    C = Zn @ Zn.T
    # chain layout: two states are ancestor-related exactly when they share a rollout
    adj = (C >= kappa) & (roll[:, None] != roll[None, :]) & (grp[:, None] == grp[None, :])
    if same_depth:
        adj &= depth[:, None] == depth[None, :]
    _, lab = connected_components(csr_matrix(adj), directed=False)
    first = {}
    for i, l in enumerate(lab):
        first.setdefault(l, i)
    return np.array([first[l] for l in lab], dtype=np.int32)


@pytest.mark.parametrize("name,groups", [("tiny", 8), ("math", 3), ("agentic", 12)])
@pytest.mark.parametrize("rule", [0, 1])
def test_classes_are_library_connected_components(oracle_mod, name, groups, rule):
    """Classes = connected components of linked comparable pairs (Sec. 4.2; scipy routine)."""
    b = W.make_batch(W.CONFIGS[name].scaled(groups))
    out = oracle_mod.run(b, {"merge_rule": rule}, want={"class_id"})
    np.testing.assert_array_equal(out["class_id"], _components(b, b["kappa"], same_depth=rule == 1))


def test_classes_match_planted_centroids(oracle_mod):
    """Generator ground truth: cross-rollout states on one centroid merge, fresh ones stay alone."""
    b = W.make_batch(W.CONFIGS["tiny"])
    out = oracle_mod.run(b, want={"class_id"})
    roll, _, grp = states_of(b)
    cid = b["planted_centroid"]
    adj = (cid[:, None] >= 0) & (cid[:, None] == cid[None, :]) & (roll[:, None] != roll[None, :]) \
        & (grp[:, None] == grp[None, :])
    _, lab = connected_components(csr_matrix(adj), directed=False)
    first = {}
    for i, l in enumerate(lab):
        first.setdefault(l, i)
    np.testing.assert_array_equal(out["class_id"], [first[l] for l in lab])
    assert 0.3 < np.mean(np.bincount(out["class_id"], minlength=len(cid))[out["class_id"]] >= 2) < 0.5


def test_permutation_equivariance(oracle_mod):
    """Reordering rollouts inside a group permutes the outputs and keeps the partition."""
    b = W.make_batch(W.CONFIGS["tiny"].scaled(2))
    so = b["rollout_step_off"]
    perm = np.concatenate([np.random.default_rng(1).permutation(8), 8 + np.random.default_rng(2).permutation(8)])
    states = np.concatenate([np.arange(so[r], so[r + 1]) for r in perm])
    pb = dict(b)
    pb["emb"] = b["emb"][states]
    pb["step_len"] = b["step_len"][states]
    pb["reward"] = b["reward"][perm]
    n = np.diff(so)[perm]
    pb["rollout_step_off"] = np.concatenate([[0], np.cumsum(n)]).astype(np.int32)
    t = np.array([b["rollout_token_off"][r + 1] - b["rollout_token_off"][r] for r in perm])
    pb["rollout_token_off"] = np.concatenate([[0], np.cumsum(t)]).astype(np.int64)
    o1 = oracle_mod.run(b)
    o2 = oracle_mod.run(pb)
    for k in ("node_score", "eta", "step_reward", "a_cor", "a_eff_node", "e_eff", "edge_adv"):
        np.testing.assert_allclose(o2[k], o1[k][states], rtol=1e-12, atol=1e-14, err_msg=k)
    # same partition: relabel both by first occurrence in the permuted order
    c1, c2 = o1["class_id"][states], o2["class_id"]
    m = {}
    for a, bb in zip(c1, c2):
        assert m.setdefault(a, bb) == bb
    assert len(set(m.values())) == len(m)


# ------------------------------------------------------------------ scores and rewards


def test_no_merge_reduces_to_grpo(oracle_mod):
    """kappa above every similarity: S is the Monte-Carlo rate (Sec. 4.3, App. G FN case),
    first-step edges get GRPO's group-normalised outcome advantage (App. B/F estimators),
    and every later edge sits in a size-1 group."""
    b = W.make_batch(W.CONFIGS["math"].scaled(4))
    out = oracle_mod.run(b, {"kappa": 2.0})
    roll, depth, _ = states_of(b)
    R = b["reward"].astype(float)
    np.testing.assert_array_equal(out["class_id"], np.arange(len(roll)))
    np.testing.assert_allclose(out["node_score"], R[roll], atol=0)
    go = b["group_rollout_off"]
    for g in range(len(go) - 1):
        rg = R[go[g]:go[g + 1]]
        assert out["root_score"][g] == pytest.approx(rg.mean(), abs=1e-15)
        grpo = (rg - rg.mean()) / (np.std(rg, ddof=1) + 1e-6)
        first = b["rollout_step_off"][go[g]:go[g + 1]]
        np.testing.assert_allclose(out["a_cor"][first], grpo, rtol=1e-12, atol=1e-12)
    later = depth >= 2
    assert np.all(out["step_reward"][later] == 0) and np.all(out["a_cor"][later] == 0)
    assert np.all(out["e_eff"] == 0) and np.all(out["eff_mask"] == 0)


def test_w0_is_tree_estimator(oracle_mod):
    """w = 0: no suffix sharing, S(v) = c_own/t_own (App. E, 'degenerates to a tree-based estimator')."""
    b = W.make_batch(W.CONFIGS["tiny"])
    out = oracle_mod.run(b, {"w": 0.0})
    roll, _, _ = states_of(b)
    np.testing.assert_allclose(out["node_score"], b["reward"][roll].astype(float), atol=0)


def test_w1_pools_whole_class(oracle_mod):
    """w = 1 with t_own = 1 everywhere: S(v) = C_Q / T_Q, the class's correct fraction."""
    b = W.make_batch(W.CONFIGS["tiny"])
    out = oracle_mod.run(b, {"w": 1.0})
    roll, _, _ = states_of(b)
    R = b["reward"][roll].astype(float)
    cid = out["class_id"]
    for q in np.unique(cid):
        mem = cid == q
        np.testing.assert_allclose(out["node_score"][mem], R[mem].mean(), rtol=1e-14)


def test_pooled_score_variance_closed_form(oracle_mod):
    """Lemma (variance with class pooling): for k merged members with one Bernoulli(p)
    terminal each, E[S] = p and Var(S) = rho p (1-p), rho = (1+(k-1)w^2)/(1+w(k-1))^2."""
    k, w, p, M = 4, 0.7, 0.3, 6000
    rng = np.random.default_rng(7)
    groups = []
    for _ in range(M):
        groups.append([([E[0] + 0.001 * E[1 + j]], [1], int(rng.random() < p)) for j in range(k)])
    b = from_rollouts(groups, kappa=0.9, w=w)
    out = oracle_mod.run(b, {"w": w}, want={"node_score", "class_id"})
    assert np.all(np.bincount(out["class_id"])[out["class_id"]] == k)
    s = out["node_score"].reshape(M, k)[:, 0]
    rho = (1 + (k - 1) * w * w) / (1 + w * (k - 1)) ** 2
    var = rho * p * (1 - p)
    assert abs(s.mean() - p) < 5 * math.sqrt(var / M)
    # standard error of a sample variance ~ var * sqrt(2/(M-1)) (a little wider for skew)
    assert abs(s.var(ddof=1) - var) < 6 * var * math.sqrt(2 / (M - 1))
    # rho is strictly below the unpooled 1 and above the fully pooled 1/k
    assert 1 / k < rho < 1


def test_all_correct_or_all_wrong(oracle_mod):
    """Constant rewards make S constant, so r_step = 0 and A_cor = 0 (Sec. 4.3-4.4);
    with all wrong the gate Sbar_Q = 0 also switches A_eff off."""
    b = W.make_batch(W.CONFIGS["tiny"])
    for val in (0, 1):
        bb = dict(b)
        bb["reward"] = np.full_like(b["reward"], val)
        out = oracle_mod.run(bb)
        assert np.all(out["node_score"] == val)
        assert np.all(out["step_reward"] == 0) and np.all(out["a_cor"] == 0)
        if val == 0:
            assert np.all(out["adv"] == 0)
        else:
            assert np.any(out["e_eff"] != 0)


# ------------------------------------------------------------------ advantages


@pytest.mark.parametrize("name,groups", [("tiny", 8), ("math", 3)])
def test_group_invariants(oracle_mod, name, groups):
    """Standardised advantages sum to zero within each correctness group and each class,
    their sample std is std/(std+eps), scores are convex combinations in [0, 1]."""
    b = W.make_batch(W.CONFIGS[name].scaled(groups))
    out = oracle_mod.run(b)
    roll, depth, grp = states_of(b)
    cid = out["class_id"]
    assert np.all((out["node_score"] >= 0) & (out["node_score"] <= 1))
    # correctness group of edge (p(v), v): the class of p(v), or the group's root
    key = np.where(depth == 1, -1 - grp, np.r_[0, cid[:-1]])
    for k in np.unique(key):
        m = key == k
        a, r = out["a_cor"][m], out["step_reward"][m]
        np.testing.assert_array_equal(out["cor_group_size"][m], m.sum())
        if m.sum() < 2:
            assert np.all(a == 0)
            continue
        assert abs(a.sum()) < 1e-9 * max(1.0, np.abs(a).max())
        sd = np.std(r, ddof=1)
        assert np.std(a, ddof=1) == pytest.approx(sd / (sd + 1e-6), rel=1e-9, abs=1e-12)
    for q in np.unique(cid):
        m = cid == q
        ae = out["a_eff_node"][m]
        if m.sum() >= 2:
            assert abs(ae.sum()) < 1e-9
            # Sbar_Q = C_Q/|Q| when every member has t_own = 1 (Eq. (combain) summed over Q)
            sbar = out["node_score"][m].mean()
            assert sbar == pytest.approx(b["reward"][roll[m]].mean(), abs=1e-13)
            # the efficiency group prefers shorter routes when Sbar_Q > 0 (App. F, path-length)
            l = depth[m]
            if sbar > 0 and l.std() > 0:
                order = np.argsort(l)
                assert np.all(np.diff(ae[order]) <= 1e-15)
        else:
            assert np.all(ae == 0)


def test_two_edge_group_closed_form(oracle_mod):
    """A correctness group of two edges standardises (ddof=1) to +-1/sqrt2 up to eps."""
    fx = golden("micro_3x2.json")
    out = oracle_mod.run(_micro_batch(fx), fx["params"])
    assert out["a_cor"][1] == pytest.approx(1 / math.sqrt(2), abs=1e-5)
    assert out["a_cor"][3] == pytest.approx(-1 / math.sqrt(2), abs=1e-5)


def test_same_depth_rule_turns_efficiency_off(oracle_mod):
    """Same-depth merging gives equal route lengths inside a class, so A_eff = 0."""
    b = W.make_batch(W.CONFIGS["tiny"])
    out = oracle_mod.run(b, {"merge_rule": 1})
    assert np.all(out["a_eff_node"] == 0) and np.all(out["e_eff"] == 0)
    _, depth, _ = states_of(b)
    cid = out["class_id"]
    assert np.all(depth == depth[cid])


def test_routes_by_path_enumeration(oracle_mod):
    """Brute force: enumerate root->state paths explicitly, find a_Q as the longest common
    prefix of the members' paths, and re-add every A_eff(v) along a_Q -> v (Sec. 4.4)."""
    b = W.make_batch(W.CONFIGS["tiny"].scaled(3))
    out = oracle_mod.run(b)
    so, go = b["rollout_step_off"], b["group_rollout_off"]
    N = len(b["step_len"])
    path = {}
    for r in range(len(so) - 1):
        for v in range(so[r], so[r + 1]):
            path[v] = ["root"] + list(range(so[r], v + 1))
    e_sum = np.zeros(N)
    cover = np.zeros(N, bool)
    cid = out["class_id"]
    for q in np.unique(cid):
        mem = list(np.nonzero(cid == q)[0])
        if len(mem) < 2:
            continue
        strict = [path[v][:-1] for v in mem]
        lcp = 0
        while all(len(p) > lcp for p in strict) and len({p[lcp] for p in strict}) == 1:
            lcp += 1
        aQ = strict[0][lcp - 1]
        assert aQ == "root"  # members of a class sit in >= 2 rollouts of a chain layout
        for v in mem:
            ell = len(path[v]) - lcp
            assert ell == len(path[v]) - 1  # l_v = depth
            for e in path[v][lcp:]:
                e_sum[e] += out["a_eff_node"][v]
                cover[e] = True
    np.testing.assert_allclose(out["e_eff"], e_sum, rtol=1e-12, atol=1e-14)
    np.testing.assert_array_equal(out["edge_eff_mask"].astype(bool), cover)


def test_token_broadcast_and_coverage(oracle_mod):
    """Every token of edge e carries A_dual(e); spans tile each rollout exactly (Sec. 4.5)."""
    b = W.make_batch(W.CONFIGS["agentic"].scaled(6))
    out = oracle_mod.run(b, {"lambda_eff": 0.5})
    want = np.repeat(out["edge_adv"], b["step_len"])
    np.testing.assert_array_equal(out["adv"], want)
    np.testing.assert_array_equal(out["adv_cor"], np.repeat(out["a_cor"], b["step_len"]))
    np.testing.assert_allclose(out["edge_adv"], out["a_cor"] + 0.5 * out["e_eff"], rtol=0, atol=0)
    assert len(out["adv"]) == b["rollout_token_off"][-1]


# ------------------------------------------------------------------ validation


def test_validation_codes(oracle_mod):
    base = W.make_batch(W.CONFIGS["tiny"].scaled(2))
    assert oracle_mod.validate(base) == 0
    bad = dict(base, reward=base["reward"].copy())
    bad["reward"][3] = 2
    assert oracle_mod.validate(bad) == 3
    bad = dict(base, step_len=base["step_len"].copy())
    bad["step_len"][5] = 0
    assert oracle_mod.validate(bad) == 2
    bad = dict(base, emb=base["emb"].copy())
    bad["emb"][7, 3] = np.nan
    assert oracle_mod.validate(bad) == 4
    bad = dict(base, rollout_token_off=base["rollout_token_off"].copy())
    bad["rollout_token_off"][4] += 1
    assert oracle_mod.validate(bad) == 2
    with pytest.raises(oracle_mod.OracleError):
        oracle_mod.run(dict(base, reward=np.full_like(base["reward"], 5)))


def test_empty_and_degenerate_groups(oracle_mod):
    """An empty prompt group, a one-rollout group and a zero embedding are all well defined."""
    grp1 = [([E[0], E[1]], [2, 3], 1)]
    grp2 = [([np.zeros(8)], [4], 0), ([E[2]], [1], 1)]
    b = from_rollouts([[], grp1, grp2], kappa=0.9)
    out = oracle_mod.run(b)
    assert len(out["adv"]) == 2 + 3 + 4 + 1
    # one rollout: root group of size 1, no advantage at all
    assert np.all(out["adv"][:5] == 0)
    # zero embedding never merges and has eta 0
    np.testing.assert_array_equal(out["class_id"][2:], [2, 3])
    assert np.all(np.isfinite(out["adv"]))


def test_threshold_is_inclusive(oracle_mod):
    """sim(u,v) >= kappa links the pair (Sec. 4.2): e1 and (1,1,1,1) have cosine exactly 1/2."""
    one = np.zeros(8)
    one[:4] = 1.0
    grp = [([E[0]], [1], 1), ([one], [1], 0), ([E[5]], [1], 0)]
    b = from_rollouts([grp], kappa=0.5)
    np.testing.assert_array_equal(oracle_mod.run(b, {"kappa": 0.5})["class_id"], [0, 0, 2])
    np.testing.assert_array_equal(oracle_mod.run(b, {"kappa": np.nextafter(0.5, 1)})["class_id"], [0, 1, 2])
