"""The seeded input generators (CPU): every shape's structure as its recipe states it,
the 1e-3 similarity margin around kappa checked by brute force on the stored values,
merges that really happen (and span depths in the branching workload), determinism in
the seed, the log-probabilities' margin from the clip bounds, and the per-layer views of
a branching batch."""
import functools

import numpy as np
import pytest
from scipy.sparse.csgraph import connected_components

from paper_2606_18954_gb300 import workloads as W

CHAIN_GROUPS = {"tiny": 8, "math": 3, "agentic": 4, "wide": 1, "full": 2}


@functools.lru_cache(maxsize=None)
def chain_batch(name):
    return W.make_batch(W.CONFIGS[name].scaled(groups=CHAIN_GROUPS[name]))


TREE_SPEC = W.TREE_CONFIGS["tree"].scaled(groups=4, d=64)


@functools.lru_cache(maxsize=None)
def tree_batch():
    return W.make_tree_batch(TREE_SPEC, seed=W.config_seed("tree"))


def emb64(b):
    e = b["emb"]
    if b["emb_dtype"] == "bf16":
        return (e.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return e.astype(np.float64)


def cosines(z):
    n = np.linalg.norm(z, axis=1)
    n[n == 0] = 1.0
    u = z / n[:, None]
    return u @ u.T


def chain_groups(b):
    go, so = b["group_rollout_off"], b["rollout_step_off"]
    for g in range(len(go) - 1):
        r0, r1 = int(go[g]), int(go[g + 1])
        s0, s1 = int(so[r0]), int(so[r1])
        roll = np.repeat(np.arange(r0, r1), np.diff(so[r0:r1 + 1]))
        yield s0, s1, roll


def tree_ancestry(par):
    """anc[i, j]: i is a strict ancestor of j (group-local parent pointers)."""
    n = len(par)
    anc = np.zeros((n, n), dtype=bool)
    for v in range(n):
        a = par[v]
        while a >= 0:
            anc[a, v] = True
            a = par[a]
    return anc


@pytest.mark.parametrize("name", sorted(CHAIN_GROUPS))
def test_chain_structure(name):
    spec, b = W.CONFIGS[name], chain_batch(name)
    G, Rg = CHAIN_GROUPS[name], spec.rollouts
    np.testing.assert_array_equal(b["group_rollout_off"], np.arange(G + 1) * Rg)
    so, sl, to = b["rollout_step_off"], b["step_len"], b["rollout_token_off"]
    n = np.diff(so)
    lo, hi = (spec.steps[1], spec.steps[1]) if spec.steps[0] == "fixed" else spec.steps[1:3]
    assert n.min() >= lo and n.max() <= hi
    assert sl.min() >= 1
    per_rollout = np.add.reduceat(sl.astype(np.int64), so[:-1])
    np.testing.assert_array_equal(np.diff(to), per_rollout)
    assert to[0] == 0
    if spec.lengths[0] == "per_step":
        assert sl.min() >= spec.lengths[1] and sl.max() <= spec.lengths[2]
    else:
        assert per_rollout.max() <= spec.lengths[3] and (per_rollout >= n).all()
    assert b["emb"].shape == (int(so[-1]), spec.d)
    assert b["emb"].dtype == (np.uint16 if spec.dtype == "bf16" else np.float32)
    assert len(b["reward"]) == G * Rg and set(np.unique(b["reward"])) <= {0, 1}
    assert np.isfinite(emb64(b)).all()


@pytest.mark.parametrize("name", sorted(CHAIN_GROUPS))
def test_chain_margin_and_merges(name):
    """No cross-rollout pair of a group lies within 1e-3 of kappa (fp64 on the stored
    values); a good share of the states do merge (shared centroids), not all."""
    b = chain_batch(name)
    kappa, margin = b["kappa"], W.CONFIGS[name].margin
    z = emb64(b)
    merged = total = 0
    for s0, s1, roll in chain_groups(b):
        C = cosines(z[s0:s1])
        cross = roll[:, None] != roll[None, :]
        assert np.abs(C[cross] - kappa).min() >= margin * (1 - 1e-9)
        ncomp, lab = connected_components(cross & (C >= kappa), directed=False)
        sizes = np.bincount(lab, minlength=ncomp)
        merged += int((sizes[lab] >= 2).sum())
        total += s1 - s0
    assert 0.2 < merged / total < 0.8, merged / total


def test_tree_structure():
    b, spec = tree_batch(), TREE_SPEC
    gs, go, gt = b["group_state_off"], b["group_rollout_off"], b["group_token_off"]
    H = len(spec.schedule)
    sl = b["step_len"]
    assert sl.min() >= spec.lengths[1] and sl.max() <= spec.lengths[2]
    for g in range(len(gs) - 1):
        s0, s1 = int(gs[g]), int(gs[g + 1])
        par = b["parent"][s0:s1]
        n = s1 - s0
        assert (par < np.arange(n)).all() and (par >= -1).all()
        kids = [[] for _ in range(n)]
        roots = []
        for v in range(n):
            (kids[par[v]] if par[v] >= 0 else roots).append(v)
        order = []  # depth-first pre-order rebuilt from the children lists

        def visit(v):
            order.append(v)
            for c in kids[v]:
                visit(c)
        for r in roots:
            visit(r)
        assert order == list(range(n))
        depth = np.zeros(n, dtype=int)
        for v in range(n):
            depth[v] = 1 if par[v] < 0 else depth[par[v]] + 1
        assert depth.max() <= H and len(roots) == spec.schedule[0]
        for v in range(n):
            assert len(kids[v]) in (0, spec.schedule[depth[v]] if depth[v] < H else 0)
        assert sum(1 for k in kids if not k) == go[g + 1] - go[g]
        assert gt[g + 1] - gt[g] == int(sl[s0:s1].astype(np.int64).sum())
        assert n <= sum(np.cumprod(spec.schedule))
    assert len(b["reward"]) == go[-1] and b["total_tokens"] == gt[-1]


def test_tree_margin_and_classes_across_depths():
    b = tree_batch()
    kappa, margin = b["kappa"], TREE_SPEC.margin
    z = emb64(b)
    gs = b["group_state_off"]
    spans_depths = 0
    for g in range(len(gs) - 1):
        s0, s1 = int(gs[g]), int(gs[g + 1])
        par = b["parent"][s0:s1]
        anc = tree_ancestry(par)
        comparable = ~(anc | anc.T) & ~np.eye(s1 - s0, dtype=bool)
        C = cosines(z[s0:s1])
        assert np.abs(C[comparable] - kappa).min() >= margin * (1 - 1e-9)
        ncomp, lab = connected_components(comparable & (C >= kappa), directed=False)
        depth = np.zeros(s1 - s0, dtype=int)
        for v in range(s1 - s0):
            depth[v] = 1 if par[v] < 0 else depth[par[v]] + 1
        for c in range(ncomp):
            if len(np.unique(depth[lab == c])) > 1:
                spans_depths += 1
    assert spans_depths > 0  # classes across depths: A_eff is not identically zero


def test_generators_are_deterministic_in_the_seed():
    spec = W.CONFIGS["tiny"].scaled(groups=2)
    a, b, c = W.make_batch(spec, seed=5), W.make_batch(spec, seed=5), W.make_batch(spec, seed=6)
    for k in ("rollout_step_off", "step_len", "emb", "reward"):
        np.testing.assert_array_equal(a[k], b[k])
    assert not np.array_equal(a["emb"], c["emb"])
    t1 = W.make_tree_batch(TREE_SPEC.scaled(groups=1), seed=9)
    t2 = W.make_tree_batch(TREE_SPEC.scaled(groups=1), seed=9)
    for k in ("parent", "step_len", "emb", "reward"):
        np.testing.assert_array_equal(t1[k], t2[k])


@pytest.mark.parametrize("clip_high", [0.2, 0.28])
def test_logprobs_keep_clear_of_the_clip_bounds(clip_high):
    lp = W.make_logprobs(200_000, 17, clip_low=0.2, clip_high=clip_high)
    for k in ("logp", "old_logp", "ref_logp"):
        assert lp[k].dtype == np.float32 and np.isfinite(lp[k]).all()
    assert (lp["old_logp"] < 0).all()
    r = np.exp(lp["logp"].astype(np.float64) - lp["old_logp"].astype(np.float64))
    for bound in (0.8, 1.0 + clip_high):
        assert np.abs(r - bound).min() >= 1e-4
    outside = np.mean((r < 0.8) | (r > 1.0 + clip_high))
    assert 0.1 < outside < 0.35, outside  # about a fifth of the tokens leave the range


@pytest.mark.parametrize("layer", [1, 2, 3, 4, 5])
def test_truncate_tree(layer):
    b = tree_batch()
    t = W.truncate_tree(b, layer)
    dep = W.tree_depths(b)
    np.testing.assert_array_equal(t["source_states"], np.nonzero(dep <= layer)[0])
    gs, tgs = b["group_state_off"], t["group_state_off"]
    for g in range(len(gs) - 1):
        s0, s1 = int(gs[g]), int(gs[g + 1])
        keep = np.nonzero(dep[s0:s1] <= layer)[0]
        assert tgs[g + 1] - tgs[g] == len(keep)
        tp = t["parent"][tgs[g]:tgs[g + 1]]
        fp = b["parent"][s0:s1]
        for i, v in enumerate(keep):  # the same parent, renumbered
            assert (tp[i] < 0) == (fp[v] < 0)
            if fp[v] >= 0:
                assert keep[tp[i]] == fp[v]
        has_child = np.zeros(s1 - s0, dtype=bool)
        has_child[fp[fp >= 0]] = True
        want = ((dep[s0:s1][keep] == layer) & has_child[keep]).astype(np.uint8)
        np.testing.assert_array_equal(t["active"][tgs[g]:tgs[g + 1]], want)
        leaves = np.ones(len(keep), dtype=bool)
        leaves[tp[tp >= 0]] = False
        assert t["group_rollout_off"][g + 1] - t["group_rollout_off"][g] == int(leaves.sum())
    assert not t["reward"].any() and len(t["reward"]) == t["group_rollout_off"][-1]
    assert t["total_tokens"] == int(t["step_len"].astype(np.int64).sum())
