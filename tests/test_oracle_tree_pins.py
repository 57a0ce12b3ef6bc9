"""Pins for the CPU oracle on the tree layout (branching rollouts, explicit
provenance parents): a hand-worked example, the equivalence with the chain
layout, the tree estimator with no merges, brute-force path enumeration for a_Q
and the routes, the paper's invariants and input validation.  CPU only."""
import json
import math
import os

import numpy as np
import pytest

from paper_2606_18954_gb300 import workloads as W

HERE = os.path.dirname(os.path.abspath(__file__))

SMALL = W.TreeSpec("small-tree", 6, (2, 3, 3), 16, "f32", 6, 0.05, 0.9, ("per_step", 1, 9),
                   ("bernoulli", 0.5), p_stop=0.2)


def golden(name):
    with open(os.path.join(HERE, "golden", name)) as f:
        return json.load(f)


def _fixture_batch(fx, root_emb=None):
    b = dict(group_rollout_off=np.asarray(fx["group_rollout_off"], np.int32),
             group_state_off=np.asarray(fx["group_state_off"], np.int32),
             group_token_off=np.asarray(fx["group_token_off"], np.int64),
             parent=np.asarray(fx["parent"], np.int32), step_len=np.asarray(fx["step_len"], np.int32),
             emb=np.asarray(fx["emb"], np.float32), emb_dtype="f32",
             reward=np.asarray(fx["reward"], np.uint8), layout="tree")
    if root_emb is not None:
        b["root_emb"] = np.asarray(root_emb, np.float32)
    return b


def _paths(parent, s0=0):
    """Root-to-state paths (lists of global state indices, "root" first) of one pre-order group."""
    path = {}
    for v in range(len(parent)):
        p = int(parent[v])
        path[s0 + v] = (["root"] if p < 0 else path[s0 + p]) + [s0 + v]
    return path


def _groups(b):
    gs = b["group_state_off"]
    return [(int(gs[g]), int(gs[g + 1])) for g in range(len(gs) - 1)]


# ------------------------------------------------------------------ worked example


def test_tree_worked_example(oracle_mod):
    """Hand-derived values of a seven-state branching graph (Sec. 4.2-4.5)."""
    fx = golden("tree_micro.json")
    p = fx["params"]
    out = oracle_mod.run(_fixture_batch(fx), p)
    eps, lam, s2 = p["std_eps"], p["lambda_eff"], math.sqrt(2.0)
    A, C, D, F, H, B, E = range(7)
    np.testing.assert_array_equal(out["class_id"], [0, 1, 2, 1, 4, 2, 6])
    np.testing.assert_allclose(out["root_score"], [0.5], rtol=1e-15)
    np.testing.assert_allclose(out["node_score"], [1 / 3, 2 / 3, 1 / 3, 1 / 3, 0, 2 / 3, 1], rtol=1e-15, atol=0)
    np.testing.assert_allclose(out["eta"], [0, 0, 0, 0, 1 / s2, 0, 0], rtol=1e-15, atol=0)
    h = (1 - 1 / s2) / 3
    r = np.array([-1 / 6, 1 / 3, 0, 0, -h, 1 / 6, 1 / 3])
    np.testing.assert_allclose(out["step_reward"], r, rtol=1e-14, atol=1e-16)
    # correctness groups: root {A,B}; class {A} -> {C,D,H}; class {D,B} -> {F,E}
    acor = np.zeros(7)
    for grp in ([A, B], [C, D, H], [F, E]):
        x = r[grp]
        sd = math.sqrt(((x - x.mean()) ** 2).sum() / (len(x) - 1))
        acor[grp] = (x - x.mean()) / (sd + eps)
    np.testing.assert_allclose(out["a_cor"], acor, rtol=1e-12, atol=1e-15)
    np.testing.assert_array_equal(out["cor_group_size"], [2, 3, 3, 2, 3, 2, 2])
    a = 0.25 / (math.sqrt(0.5) + eps)
    np.testing.assert_allclose(out["a_eff_node"], [0, a, -a, -a, 0, a, 0], rtol=1e-14, atol=0)
    e_eff = np.array([-a, a, -2 * a, -a, 0, a, 0])
    np.testing.assert_allclose(out["e_eff"], e_eff, rtol=1e-14, atol=0)
    np.testing.assert_array_equal(out["edge_eff_mask"], [1, 1, 1, 1, 0, 1, 0])
    np.testing.assert_allclose(out["edge_adv"], acor + lam * e_eff, rtol=1e-14, atol=1e-15)
    # every edge's tokens once, in state order (Sec. 4.5 sums over direct edges)
    np.testing.assert_array_equal(out["adv"], np.repeat(out["edge_adv"], fx["step_len"]))
    np.testing.assert_array_equal(out["eff_mask"], np.repeat([1, 1, 1, 1, 0, 1, 0], fx["step_len"]))


def test_tree_root_embedding_variant(oracle_mod):
    """A prompt embedding gives eta on root edges: root_emb = e3 makes eta(root, B) = 1."""
    fx = golden("tree_micro.json")
    out = oracle_mod.run(_fixture_batch(fx, fx["root_emb_variant"]), fx["params"])
    eps = fx["params"]["std_eps"]
    np.testing.assert_allclose(out["eta"][[0, 5]], [0.0, 1.0], atol=1e-15)
    v = (1 / 12) / (math.sqrt(2) / 12 + eps)
    np.testing.assert_allclose(out["a_cor"][[0, 5]], [-v, v], rtol=1e-12)


def test_tree_eta_is_clamped_at_zero(oracle_mod):
    """eta = max(0, sim) (Sec. 4.3): with E's embedding anti-parallel to its parent B
    (cosine -1) eta(B, E) is 0, not -1, so r(E) = S(E) - S(B) = 1 - 2/3 = 1/3 (the
    unclamped value would double it); no other link changes (E is orthogonal to the
    others and anti-parallel to D, which stays unmerged)."""
    fx = golden("tree_micro.json")
    b = _fixture_batch(fx)
    b["emb"] = b["emb"].copy()
    b["emb"][6] = -b["emb"][5]
    out = oracle_mod.run(b, fx["params"])
    assert out["eta"][6] == 0.0
    assert out["step_reward"][6] == pytest.approx(1.0 / 3.0, abs=1e-15)
    np.testing.assert_array_equal(out["class_id"], [0, 1, 2, 1, 4, 2, 6])


# ------------------------------------------------------------------ chain layout as a tree


@pytest.mark.parametrize("name,groups", [("tiny", 8), ("math", 2), ("agentic", 8)])
@pytest.mark.parametrize("rule", [0, 1])
def test_chain_written_as_tree_is_identical(oracle_mod, name, groups, rule):
    """A chain-layout batch and the same rollouts given as provenance parents describe the
    same graph: every output is identical, tokens included."""
    b = W.make_batch(W.CONFIGS[name].scaled(groups))
    t = W.as_tree(b)
    assert oracle_mod.validate(t) == 0
    x = oracle_mod.run(b, {"merge_rule": rule})
    y = oracle_mod.run(t, {"merge_rule": rule})
    for k in x:
        np.testing.assert_array_equal(x[k], y[k], err_msg=k)


# ------------------------------------------------------------------ closed forms and brute force


def test_tree_no_merge_is_subtree_success_rate(oracle_mod):
    """With no merges (kappa > 1) or w = 0, S(v) is the fraction of correct leaves among the
    leaves reachable from v (Eq. (combain) with Q(v) = {v}), counted here by enumerating
    every root-to-leaf path."""
    b = W.make_tree_batch(SMALL, seed=11)
    for params in ({"kappa": 2.0}, {"w": 0.0}):
        out = oracle_mod.run(b, params)
        go = b["group_rollout_off"]
        for g, (s0, s1) in enumerate(_groups(b)):
            path = _paths(b["parent"][s0:s1], s0)
            leaves = [v for v in range(s0, s1) if not any(int(b["parent"][u]) + s0 == v for u in range(s0, s1)
                                                         if b["parent"][u] >= 0)]
            assert len(leaves) == go[g + 1] - go[g]
            rew = {v: int(b["reward"][go[g] + k]) for k, v in enumerate(leaves)}
            for v in range(s0, s1):
                below = [z for z in leaves if v in path[z]]
                assert out["node_score"][v] == pytest.approx(sum(rew[z] for z in below) / len(below), abs=1e-15)
            assert out["root_score"][g] == pytest.approx(sum(rew.values()) / len(leaves), abs=1e-15)


def test_tree_aQ_and_routes_by_path_enumeration(oracle_mod):
    """Brute force: a_Q is the longest common prefix of the members' strict-ancestor paths,
    l_v the number of edges after it; A_eff(v) (z-score of -l over Q, gated by the mean
    score) is added to every edge of a_Q -> v (Sec. 4.4)."""
    b = W.make_tree_batch(SMALL.scaled(10), seed=12)
    out = oracle_mod.run(b)
    N = len(b["step_len"])
    e_sum, cover = np.zeros(N), np.zeros(N, bool)
    deeper = 0
    for s0, s1 in _groups(b):
        path = _paths(b["parent"][s0:s1], s0)
        cid = out["class_id"][s0:s1]
        for q in np.unique(cid):
            mem = [s0 + int(i) for i in np.nonzero(cid == q)[0]]
            if len(mem) < 2:
                continue
            strict = [path[v][:-1] for v in mem]
            lcp = 0
            while all(len(p) > lcp for p in strict) and len({p[lcp] for p in strict}) == 1:
                lcp += 1
            deeper += lcp > 1
            ell = np.array([len(path[v]) - lcp for v in mem], float)
            x = -ell
            sd = math.sqrt(((x - x.mean()) ** 2).sum() / (len(x) - 1))
            sbar = np.mean(out["node_score"][mem])
            for k, v in enumerate(mem):
                A = sbar * (x[k] - x.mean()) / (sd + 1e-6)
                assert out["a_eff_node"][v] == pytest.approx(A, rel=1e-12, abs=1e-14)
                for e in path[v][lcp:]:
                    e_sum[e] += A
                    cover[e] = True
    assert deeper > 0  # some class's deepest shared predecessor lies below the root
    np.testing.assert_allclose(out["e_eff"], e_sum, rtol=1e-12, atol=1e-13)
    np.testing.assert_array_equal(out["edge_eff_mask"].astype(bool), cover)


def test_tree_classes_are_components_of_non_causal_links(oracle_mod):
    """Classes = connected components of the comparable pairs (no ancestor relation) with
    cosine >= kappa, found here with scipy; label = smallest member."""
    from scipy.sparse import csr_matrix
    from scipy.sparse.csgraph import connected_components
    b = W.make_tree_batch(SMALL.scaled(8), seed=13)
    out = oracle_mod.run(b)
    z = b["emb"].astype(np.float64)
    for s0, s1 in _groups(b):
        path = _paths(b["parent"][s0:s1], s0)
        n = s1 - s0
        zz = z[s0:s1] / np.linalg.norm(z[s0:s1], axis=1, keepdims=True)
        C = zz @ zz.T
        anc = np.zeros((n, n), bool)
        for v in range(n):
            for u in path[s0 + v][1:-1]:
                anc[u - s0, v] = anc[v, u - s0] = True
        adj = (C >= b["kappa"]) & ~anc & ~np.eye(n, dtype=bool)
        _, lab = connected_components(csr_matrix(adj), directed=False)
        first = {}
        want = np.array([first.setdefault(l, s0 + i) for i, l in enumerate(lab)])
        np.testing.assert_array_equal(out["class_id"][s0:s1], want)


def test_tree_invariants(oracle_mod):
    """S in [0,1]; every correctness group (key = class of p(v)) has zero-sum A_cor and
    sample std std/(std+eps); every class's A_eff sums to 0; same-depth merging turns
    A_eff off (all members of a class then share l_v)."""
    b = W.make_tree_batch(W.TREE_CONFIGS["tree"].scaled(3))
    out = oracle_mod.run(b)
    assert np.all((out["node_score"] >= 0) & (out["node_score"] <= 1))
    for s0, s1 in _groups(b):
        par = b["parent"][s0:s1]
        cid = out["class_id"][s0:s1]
        key = np.where(par < 0, -1, cid[np.maximum(par, 0)])
        for k in np.unique(key):
            m = np.nonzero(key == k)[0] + s0
            if len(m) >= 2:
                assert abs(out["a_cor"][m].sum()) < 1e-9
                assert out["cor_group_size"][m[0]] == len(m)
        for q in np.unique(cid):
            m = np.nonzero(cid == q)[0] + s0
            if len(m) >= 2:
                assert abs(out["a_eff_node"][m].sum()) < 1e-9
    same = oracle_mod.run(b, {"merge_rule": 1})
    assert np.all(same["e_eff"] == 0)
    depth = np.zeros(len(b["parent"]), int)
    for s0, s1 in _groups(b):
        for v in range(s0, s1):
            p = b["parent"][v]
            depth[v] = 1 if p < 0 else depth[s0 + p] + 1
    for q in np.unique(same["class_id"]):
        assert len(set(depth[same["class_id"] == q])) == 1


def test_tree_sibling_order_equivariance(oracle_mod):
    """Listing the root's subtrees in another order (still a pre-order) permutes every
    per-state output and leaves the class partition unchanged."""
    b = W.make_tree_batch(SMALL.scaled(1), seed=14)
    n = len(b["parent"])
    par = b["parent"]
    tops = [v for v in range(n) if par[v] < 0]
    ends = tops[1:] + [n]
    blocks = [list(range(a, e)) for a, e in zip(tops, ends)][::-1]
    perm = np.array([v for blk in blocks for v in blk])  # new position -> old state
    inv = np.empty(n, int)
    inv[perm] = np.arange(n)
    newpar = np.array([-1 if par[v] < 0 else inv[par[v]] for v in perm], np.int32)
    leaves_old = [v for v in range(n) if v not in set(par.tolist())]
    leaves_new = [v for v in range(n) if v not in set(newpar.tolist())]
    rew_of = dict(zip(leaves_old, b["reward"]))
    nb = dict(b, parent=newpar, emb=b["emb"][perm], step_len=b["step_len"][perm],
              reward=np.array([rew_of[perm[v]] for v in leaves_new], np.uint8))
    x, y = oracle_mod.run(b), oracle_mod.run(nb)
    for k in ("node_score", "step_reward", "a_cor", "e_eff", "edge_adv", "edge_eff_mask"):
        np.testing.assert_allclose(y[k], x[k][perm], rtol=1e-12, atol=1e-14, err_msg=k)
    same = y["class_id"][:, None] == y["class_id"][None, :]
    np.testing.assert_array_equal(same, (x["class_id"][perm][:, None] == x["class_id"][perm][None, :]))


# ------------------------------------------------------------------ validation


def test_tree_validation_codes(oracle_mod):
    fx = golden("tree_micro.json")
    base = _fixture_batch(fx)
    assert oracle_mod.validate(base) == 0

    def with_(**kw):
        return dict(base, **{k: np.asarray(v, base[k].dtype) for k, v in kw.items()})

    assert oracle_mod.validate(with_(parent=[-1, 0, 0, 2, 0, -1, 7])) == 2   # parent after the state
    assert oracle_mod.validate(with_(parent=[-1, 0, 0, 3, 0, -1, 5])) == 2   # parent is the state itself
    assert oracle_mod.validate(with_(parent=[-1, 0, 0, 2, 0, -1, -2])) == 2  # below -1
    # F moved under C while D sits between them: C's subtree is no longer contiguous
    assert oracle_mod.validate(with_(parent=[-1, 0, 0, 1, 0, -1, 5])) == 2
    # the same parents as a valid pre-order have one leaf fewer: the leaf count must match
    assert oracle_mod.validate(with_(parent=[-1, 0, 1, 2, 0, -1, 5])) == 2
    assert oracle_mod.validate(with_(group_token_off=[0, 18])) == 2
    assert oracle_mod.validate(with_(step_len=[3, 2, 0, 4, 2, 5, 2])) == 2
    assert oracle_mod.validate(with_(reward=[1, 0, 2, 1])) == 3
    bad = with_()
    bad["emb"] = bad["emb"].copy()
    bad["emb"][2, 0] = np.inf
    assert oracle_mod.validate(bad) == 4
