"""Tree layout (branching rollouts with explicit provenance parents) on the GPU,
through the C ABI, against the CPU oracle element by element.

Same bar as the chain layout: class ids bit-exact; every fp32 output within
|gpu - ref| <= 1e-5 |ref| + 1e-6 of the oracle's fp64 value rounded to fp32.
Covers the three similarity paths (fused group-resident kernel, tiled tensor-core
path, CUDA-core path), both merge rules, the paper's branching schedules
(including one whose groups exceed the fused kernel's 384 states), a chain batch
written as a tree, prompt embeddings, degenerate shapes, every device-side error
of the layout and the full-size tree workload on sampled groups.
"""
import functools

import numpy as np
import pytest

from paper_2606_18954_gb300 import workloads as W
from test_gpu_parity import (PATH_FLAGS, assert_close, batch_of, compare, gp_mod, oracle_params,  # noqa: F401
                             oracle_run, run_gpu, torch_cuda)

pytestmark = pytest.mark.gpu

KAPPA = 0.9


@functools.lru_cache(maxsize=None)
def tree_of(name, groups=None, seed=None, **kw):
    spec = W.TREE_CONFIGS[name] if name in W.TREE_CONFIGS else SPECS[name]
    if seed is None and name not in W.TREE_CONFIGS:
        seed = W.BASE_SEED + 100 + sorted(SPECS).index(name)
    if groups is not None or kw:
        spec = spec.scaled(groups, **kw)
    return W.make_tree_batch(spec, seed=seed)


# Branching schedules of the paper's branching study (b_1..b_H children per active state),
# at d = 64 so that the oracle stays quick; {7,6,5,4,3} gives groups of ~2500 states (tiled path).
SPECS = {
    "sched4532": W.TreeSpec("sched4532", 3, (4, 5, 3, 2), 64, "bf16", 8, 0.05, KAPPA, ("per_step", 8, 96),
                            ("bernoulli", 0.5)),
    "sched54222": W.TreeSpec("sched54222", 3, (5, 4, 2, 2, 2), 64, "bf16", 8, 0.05, KAPPA, ("per_step", 8, 96),
                             ("beta", 2.0, 2.0)),
    "sched243222": W.TreeSpec("sched243222", 2, (2, 4, 3, 2, 2, 2), 64, "bf16", 8, 0.05, KAPPA,
                              ("per_step", 8, 96), ("bernoulli", 0.3)),
    "sched76543": W.TreeSpec("sched76543", 1, (7, 6, 5, 4, 3), 64, "bf16", 16, 0.05, KAPPA, ("per_step", 4, 40),
                             ("bernoulli", 0.5)),
    "small_f32": W.TreeSpec("small_f32", 6, (2, 3, 3), 32, "f32", 6, 0.05, KAPPA, ("per_step", 1, 9),
                            ("bernoulli", 0.5), p_stop=0.2),
}


def tree_margin_ok(b, kappa, margin=1e-3):
    """No comparable pair (not ancestor-related, same group) within `margin` of kappa."""
    from batches import emb_f64
    Z = emb_f64(b)
    gs, par = b["group_state_off"], b["parent"]
    for g in range(len(gs) - 1):
        s0, s1 = int(gs[g]), int(gs[g + 1])
        n = s1 - s0
        if n < 2:
            continue
        end = W.subtree_end(par[s0:s1])
        idx = np.arange(n)
        comp = (idx[None, :] >= end[:, None]) | (idx[:, None] >= end[None, :])
        X = Z[s0:s1]
        nr = np.linalg.norm(X, axis=1)
        nz = nr > 0
        Xn = X / np.where(nz, nr, 1.0)[:, None]
        C = Xn @ Xn.T
        m = comp & nz[:, None] & nz[None, :]
        if np.any(np.abs(C[m] - kappa) < margin):
            return False
    return True


def tree_from_groups(groups, d, dtype="bf16", kappa=KAPPA, rng=None):
    """A tree-layout batch from hand-built groups: each group is (parent list, emb rows, rewards of its
    leaves in state order, step lengths)."""
    go, gs, gt, par, sl, emb, rew = [0], [0], [0], [], [], [], []
    for parent, rows, rewards, lens in groups:
        par.extend(parent)
        emb.extend(rows)
        rew.extend(rewards)
        sl.extend(lens)
        go.append(go[-1] + len(rewards))
        gs.append(gs[-1] + len(parent))
        gt.append(gt[-1] + int(np.sum(lens)))
    e = np.asarray(emb, np.float64).reshape(-1, d).astype(np.float32)
    if dtype == "bf16":
        e = W.f32_to_bf16_bits(e)
    return dict(group_rollout_off=np.asarray(go, np.int32), group_state_off=np.asarray(gs, np.int32),
                group_token_off=np.asarray(gt, np.int64), total_tokens=gt[-1],
                parent=np.asarray(par, np.int32), step_len=np.asarray(sl, np.int32), emb=e, emb_dtype=dtype,
                reward=np.asarray(rew, np.uint8), kappa=kappa, w=0.7, lambda_eff=1.0, layout="tree")


def _leaves(parent):
    n = len(parent)
    has_child = np.zeros(n, bool)
    for p in parent:
        if p >= 0:
            has_child[p] = True
    return int(np.sum(~has_child))


def _rows(rng, n, d, share=None, dirs=None):
    out = []
    for i in range(n):
        k = share(i) if share else None
        if k is None:
            out.append(rng.standard_normal(d))
        else:
            out.append(dirs[k] + 0.01 * rng.standard_normal(d) / np.sqrt(d))
    return out


def shape_group(kind, rng, d=64):
    """Degenerate and boundary-size tree groups."""
    dirs = rng.standard_normal((6, d))
    if kind == "path":        # one rollout of 300 steps: nothing is comparable
        parent = [-1] + list(range(299))
    elif kind == "star":      # 200 single-step rollouts: every pair comparable
        parent = [-1] * 200
    elif kind == "single":    # one state
        parent = [-1]
    elif kind == "broom":     # a 40-step handle, then 60 leaves under its end
        parent = [-1] + list(range(39)) + [39] * 60
    elif kind == "binary":    # complete binary tree of depth 8 (510 states), pre-order
        parent = []

        def add(p, depth):
            v = len(parent)
            parent.append(p)
            if depth < 8:
                add(v, depth + 1)
                add(v, depth + 1)
        add(-1, 1)
        add(-1, 1)
    elif kind == "n384":      # 384 states: 16 root children, each a path of 24
        parent = []
        for _ in range(16):
            parent.append(-1)
            parent.extend(range(len(parent) - 1, len(parent) + 22))
    else:
        raise KeyError(kind)
    n = len(parent)
    depth = np.zeros(n, int)
    for v in range(n):
        depth[v] = 1 if parent[v] < 0 else depth[parent[v]] + 1
    rows = _rows(rng, n, d, share=lambda i: (depth[i] % 3) if (i * 7) % 5 == 0 else None, dirs=dirs)
    lens = list(rng.integers(1, 30, size=n))
    rewards = list(rng.integers(0, 2, size=_leaves(parent)))
    return parent, rows, rewards, lens


def flags_for(b, path):
    if path != "simt" and b["emb_dtype"] != "bf16":
        pytest.skip("fp32 embeddings always use the CUDA-core similarity kernel")
    return PATH_FLAGS[path]


PATHS = pytest.mark.parametrize("path", ["fused", "tiled", "simt"])


# ------------------------------------------------------------------ parity


@PATHS
@pytest.mark.parametrize("rule", [0, 1])
def test_tree_parity_scaled(gp_mod, path, rule):
    """The tree workload (schedule {2,5,4,2,2}, bf16 d=1024) on 6 groups."""
    b = tree_of("tree", 6)
    params = oracle_params(b, merge_rule=rule)
    ref = oracle_run(b, params)
    assert np.any(ref["edge_eff_mask"]) and np.any(ref["class_id"] != np.arange(len(ref["class_id"])))
    compare(run_gpu(gp_mod, b, params, flags=flags_for(b, path)), ref, f"tree/{rule}/{path}")


@pytest.mark.parametrize("sched", ["sched4532", "sched54222", "sched243222", "small_f32"])
@PATHS
def test_tree_parity_schedules(gp_mod, sched, path):
    b = tree_of(sched)
    params = oracle_params(b)
    compare(run_gpu(gp_mod, b, params, flags=flags_for(b, path)), oracle_run(b, params), f"{sched}/{path}")


@pytest.mark.parametrize("path", ["fused", "simt"])
def test_tree_parity_wide_schedule(gp_mod, path):
    """{7,6,5,4,3}: one group of ~2500 states (above the fused kernel's 384, so the default
    launch takes the tiled tensor-core path)."""
    b = tree_of("sched76543")
    assert int(np.diff(b["group_state_off"]).max()) > 384
    params = oracle_params(b)
    compare(run_gpu(gp_mod, b, params, flags=flags_for(b, path)), oracle_run(b, params), f"sched76543/{path}")


@pytest.mark.parametrize("name,groups", [("math", 3), ("agentic", 8), ("tiny", 3)])
@PATHS
def test_chain_written_as_tree(gp_mod, name, groups, path):
    """A chain batch in the tree layout gives the chain oracle's results (tokens stay in place)."""
    b = batch_of(name, groups)
    t = W.as_tree(b)
    params = oracle_params(b)
    compare(run_gpu(gp_mod, t, params, flags=flags_for(t, path)), oracle_run(b, params), f"{name} as tree/{path}")


@PATHS
def test_tree_root_embedding(gp_mod, path):
    b = dict(tree_of("tree", 3))
    rng = np.random.default_rng(9)
    gs = b["group_state_off"]
    first = gs[:-1]
    base = W.bf16_bits_to_f32(b["emb"][first]).astype(np.float64)
    root = base + 0.5 * rng.standard_normal(base.shape) / np.sqrt(base.shape[1])
    b["root_emb"] = W.f32_to_bf16_bits(root.astype(np.float32))
    params = oracle_params(b)
    ref = oracle_run(b, params)
    assert np.any(ref["eta"][first] > 0)
    compare(run_gpu(gp_mod, b, params, flags=flags_for(b, path)), ref, f"tree root_emb/{path}")


@PATHS
def test_tree_shapes(gp_mod, path):
    """Path, star, single state, broom, complete binary tree (510 states), 384 states, and empty
    groups in between."""
    rng = np.random.default_rng(77)
    kinds = ["path", "star", "single", "broom", "n384"] + ([] if path == "fused" else ["binary"])
    groups = []
    for k in kinds:
        groups.append(shape_group(k, rng))
        groups.append(([], [], [], []))  # an empty prompt group
    b = tree_from_groups(groups, 64)
    assert tree_margin_ok(b, KAPPA)
    params = oracle_params(b)
    ref = oracle_run(b, params)
    compare(run_gpu(gp_mod, b, params, flags=flags_for(b, path)), ref, f"shapes/{path}")


@pytest.mark.parametrize("path", ["fused", "tiled"])
def test_tree_binary_default_launch(gp_mod, path):
    """A 510-state group with 384-state groups: the default launch takes the tiled path."""
    rng = np.random.default_rng(78)
    b = tree_from_groups([shape_group("binary", rng), shape_group("n384", rng)], 64)
    assert tree_margin_ok(b, KAPPA)
    params = oracle_params(b)
    compare(run_gpu(gp_mod, b, params, flags=0 if path == "fused" else 2), oracle_run(b, params), "binary")


@pytest.mark.parametrize("path", ["fused", "tiled"])
def test_tree_deterministic(gp_mod, path):
    b = tree_of("tree", 4)
    params = oracle_params(b)
    a1 = run_gpu(gp_mod, b, params, flags=PATH_FLAGS[path])
    a2 = run_gpu(gp_mod, b, params, flags=PATH_FLAGS[path])
    for k in a1:
        np.testing.assert_array_equal(a1[k], a2[k], err_msg=k)


@pytest.mark.parametrize("path", ["fused", "tiled"])
def test_tree_full_size_whole_batch(gp_mod, path):
    """The whole tree workload (128 prompts, schedule {2,5,4,2,2}, bf16 d=1024) in the
    benchmark's launch configuration (fused) and on the tiled path, every output of every
    group against the oracle."""
    b = tree_of("tree")
    params = oracle_params(b)
    gpu = run_gpu(gp_mod, b, params, flags=PATH_FLAGS[path])
    compare(gpu, oracle_run(b, params, threads=16), f"tree whole batch/{path}")
    np.testing.assert_array_equal(gpu["adv"], np.repeat(gpu["edge_adv"], b["step_len"]))
    assert np.all((gpu["node_score"] >= 0) & (gpu["node_score"] <= 1))


# ------------------------------------------------------------------ errors


def _expect(P, b, code, flags):
    import torch
    gp = P.GraphPO(kappa=KAPPA, flags=flags)
    db = P.Batch.from_arrays(b, device="cuda")
    gp(db)
    with pytest.raises(P.GraphPOError) as e:
        gp.check()
    assert e.value.code == code, gp.last_error()
    ok = P.Batch.from_arrays(tree_of("tree", 2), device="cuda")
    gp2 = P.GraphPO(kappa=0.92, flags=flags)
    gp2(ok)
    gp2.check()
    torch.cuda.synchronize()


def _bad(kind):
    b = {k: (v.copy() if isinstance(v, np.ndarray) else v) for k, v in tree_of("tree", 3).items()}
    gs = b["group_state_off"]
    s0 = int(gs[1])
    if kind == "parent_ahead":        # a parent that is not an earlier state
        b["parent"][s0 + 3] = 5
    elif kind == "not_preorder":      # a state after the first root child's subtree hung under it
        p = b["parent"]
        end0 = int(W.subtree_end(p[s0:int(gs[2])])[0])  # group-local end of state 0's subtree
        v = s0 + end0 + 1              # its predecessor v - 1 lies outside that subtree
        assert v < int(gs[2])
        p[v] = 0                       # state 0 is then not on the path from the root to v - 1
    elif kind == "leaf_count":        # one reward too many for the group's leaves
        b["group_rollout_off"] = b["group_rollout_off"].copy()
        b["group_rollout_off"][1] += 1
        b["group_rollout_off"][2:] += 1
        b["reward"] = np.concatenate([b["reward"], [0]]).astype(np.uint8)
    elif kind == "reward":
        b["reward"][4] = 2
    elif kind == "tokens":
        b["group_token_off"][2] += 1
    elif kind == "step_len":
        b["step_len"][s0 + 2] = 0
    return b


@pytest.mark.parametrize("kind,code", [("parent_ahead", 2), ("not_preorder", 2), ("leaf_count", 2), ("reward", 3),
                                       ("tokens", 2), ("step_len", 2)])
@pytest.mark.parametrize("path", ["fused", "tiled"])
def test_tree_errors(gp_mod, kind, code, path):
    _expect(gp_mod, _bad(kind), code, PATH_FLAGS[path])
