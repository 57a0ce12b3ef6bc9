"""Seeded synthetic rollout-group batches shaped like GraphPO's training workloads.

This module only draws inputs. It holds none of the method's arithmetic: it
produces step boundaries, step lengths, state embeddings and binary rewards,
and nothing downstream of them (no classes, scores, rewards or advantages).

Layout of a batch ("chain layout": every rollout is a chain root -> s_1 -> ... ->
s_{n_r}; state (r, h) is the node reached after generated step h, and the step
itself is the direct edge entering it, GraphPO Sec. 4.2):

  group_rollout_off  int32 [G+1]  rollouts of prompt group g are [off[g], off[g+1])
  rollout_step_off   int32 [R+1]  states of rollout r are [off[r], off[r+1])
  step_len           int32 [N]    tokens of the step entering each state
  rollout_token_off  int64 [R+1]  packed token span of each rollout
  emb                [N, d]       state embeddings z_v, bf16 bit patterns (uint16)
                                  or float32
  reward             uint8 [R]    verifier reward R(z) in {0, 1} of each rollout

Tree layout (`make_tree_batch`: branching rollouts expanded layer by layer
with a branching schedule b_1..b_H, GraphPO Sec. 4.2 and its branching-schedule
study): each group's states are listed in depth-first pre-order and

  group_rollout_off  int32 [G+1]  the group's leaves (terminal states) = its rollouts
  group_state_off    int32 [G+1]  states of group g are [off[g], off[g+1])
  parent             int32 [N]    group-local index of p(v); -1 for the prompt root
  step_len           int32 [N]    tokens of the edge entering each state
  group_token_off    int64 [G+1]  every edge's tokens once, in state order
  reward             uint8 [R]    verifier reward of each leaf, leaves in state order

Recipe per config (seed 20261202 + k, numpy default_rng, drawn group by group,
rollout by rollout, step by step):
  * every prompt group owns K unit centroids (Gaussian, normalised);
  * a state is "shared" with probability p_share; a shared state at step h
    (1-based) takes centroid  floor((h-1) K / n_max) + U{-1,0,1}  (mod K), so
    states of nearby depth in different rollouts land on the same centroid;
    otherwise it is a fresh random unit direction;
  * isotropic noise of total norm ~sigma (sigma/sqrt(d) per coordinate) is added
    and the row is rounded to bf16 (round-to-nearest-even), fp32 for `tiny`;
  * margin filter: any state with a cross-rollout cosine (computed in fp64 on the
    rounded values) within `margin` of kappa is redrawn until none is left, so
    that the threshold decision is unambiguous at any reasonable precision.
Trees: the root expands b_1 children; a state at layer h < H ends its branch
early with probability p_stop, else expands b_{h+1} children; states of layer H
are terminal.  Structure first (pre-order), then step lengths, embeddings (the
same centroid recipe with n_max = max(H, K/2): the band advances by at most two
centroids per layer, so neighbouring layers share centroids and classes span
depths, as in the chain workloads), leaf rewards and the margin filter over the
pairs not in an ancestor-descendant relation.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import numpy as np

BASE_SEED = 20261202


@dataclasses.dataclass(frozen=True)
class Spec:
    name: str
    groups: int
    rollouts: int                 # rollouts per prompt group
    d: int
    dtype: str                    # "bf16" | "f32"
    centroids: int
    sigma: float
    kappa: float
    # steps per rollout: ("fixed", n) | ("uniform", lo, hi)
    steps: tuple
    # token lengths: ("per_step", lo, hi)  each step U[lo, hi]
    #                ("lognormal", median, sigma_ln, cap)  whole response, then cut
    lengths: tuple
    # rewards: ("bernoulli", p) | ("beta", a, b)  p_g ~ Beta(a, b) per prompt
    rewards: tuple
    p_share: float = 0.48
    margin: float = 1e-3
    w: float = 0.7
    lambda_eff: float = 1.0

    def scaled(self, groups: Optional[int] = None, **kw) -> "Spec":
        """Same distribution with fewer groups (or other overrides)."""
        if groups is not None:
            kw["groups"] = groups
        return dataclasses.replace(self, **kw)


# The five workload shapes: tiny, math RLVR, agentic search, wide groups, full batch.
CONFIGS = {
    "tiny": Spec("tiny", 8, 8, 256, "f32", 12, 0.05, 0.90,
                 ("fixed", 6), ("per_step", 32, 256), ("bernoulli", 0.5)),
    "math": Spec("math", 128, 16, 1024, "bf16", 32, 0.08, 0.92,
                 ("uniform", 12, 20), ("lognormal", 2048, 0.5, 8192), ("beta", 2.0, 2.0)),
    "agentic": Spec("agentic", 256, 8, 1024, "bf16", 16, 0.08, 0.92,
                    ("uniform", 4, 10), ("per_step", 64, 1024), ("bernoulli", 0.3)),
    "wide": Spec("wide", 64, 64, 2048, "bf16", 64, 0.06, 0.92,
                 ("fixed", 32), ("per_step", 32, 512), ("bernoulli", 0.5)),
    "full": Spec("full", 512, 16, 1024, "bf16", 48, 0.08, 0.92,
                 ("uniform", 15, 25), ("lognormal", 4096, 0.5, 16384), ("beta", 1.0, 1.0)),
}
CONFIG_ORDER = ["tiny", "math", "agentic", "wide", "full"]


@dataclasses.dataclass(frozen=True)
class TreeSpec:
    name: str
    groups: int
    schedule: tuple               # b_1..b_H: children of every expanded state of layer h-1
    d: int
    dtype: str                    # "bf16" | "f32"
    centroids: int
    sigma: float
    kappa: float
    lengths: tuple                # ("per_step", lo, hi): each edge U[lo, hi] tokens
    rewards: tuple                # as Spec.rewards
    p_stop: float = 0.1           # a state above the last layer ends its branch early
    p_share: float = 0.48
    margin: float = 1e-3
    w: float = 0.7
    lambda_eff: float = 1.0

    def scaled(self, groups: Optional[int] = None, **kw) -> "TreeSpec":
        if groups is not None:
            kw["groups"] = groups
        return dataclasses.replace(self, **kw)


# Branching rollouts with the schedule {2,5,4,2,2} (the best of the paper's branching
# study): at most 2 + 10 + 40 + 80 + 160 = 292 states and 160 leaves per prompt.
TREE_CONFIGS = {
    "tree": TreeSpec("tree", 128, (2, 5, 4, 2, 2), 1024, "bf16", 32, 0.08, 0.92,
                     ("per_step", 64, 512), ("beta", 2.0, 2.0)),
}


def config_seed(name: str) -> int:
    if name in TREE_CONFIGS:
        return BASE_SEED + len(CONFIG_ORDER) + list(TREE_CONFIGS).index(name)
    return BASE_SEED + CONFIG_ORDER.index(name)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bfloat16 (nearest-even) and return the uint16 bit patterns."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return u.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (b.astype(np.uint32) << 16).view(np.float32)


def _n_steps(rng, spec: Spec) -> int:
    if spec.steps[0] == "fixed":
        return int(spec.steps[1])
    lo, hi = spec.steps[1], spec.steps[2]
    return int(rng.integers(lo, hi + 1))


def _max_steps(spec: Spec) -> int:
    return int(spec.steps[1] if spec.steps[0] == "fixed" else spec.steps[2])


def _lengths(rng, spec: Spec, n: int) -> np.ndarray:
    if spec.lengths[0] == "per_step":
        lo, hi = spec.lengths[1], spec.lengths[2]
        return rng.integers(lo, hi + 1, size=n).astype(np.int32)
    median, s_ln, cap = spec.lengths[1], spec.lengths[2], spec.lengths[3]
    total = int(round(rng.lognormal(math.log(median), s_ln)))
    total = max(n, min(cap, total))
    if n == 1:
        return np.array([total], dtype=np.int32)
    cuts = np.sort(rng.choice(np.arange(1, total), size=n - 1, replace=False))
    edges = np.concatenate([[0], cuts, [total]])
    return np.diff(edges).astype(np.int32)


def _unit(rng, k: int, d: int) -> np.ndarray:
    v = rng.standard_normal((k, d))
    return v / np.linalg.norm(v, axis=1, keepdims=True)


def _draw_states(rng, spec: Spec, cents: np.ndarray, depth: np.ndarray, n_max: int):
    """Embeddings (float64, before rounding) and planted centroids (-1 = fresh) for states at `depth`."""
    n, d, K = len(depth), spec.d, cents.shape[0]
    share = rng.random(n) < spec.p_share
    jitter = rng.integers(-1, 2, size=n)
    fresh = _unit(rng, n, d) if n else np.zeros((0, d))
    noise = rng.standard_normal((n, d)) * (spec.sigma / math.sqrt(d))
    band = ((depth - 1) * K) // n_max
    cid = np.where(share, (band + jitter) % K, -1).astype(np.int32)
    base = np.where(share[:, None], cents[np.maximum(cid, 0)], fresh)
    return base + noise, cid


def _round(spec: Spec, z: np.ndarray):
    """Rounded storage form and its exact float64 value."""
    if spec.dtype == "bf16":
        bits = f32_to_bf16_bits(z.astype(np.float32))
        return bits, bf16_bits_to_f32(bits).astype(np.float64)
    f = z.astype(np.float32)
    return f, f.astype(np.float64)


def make_batch(spec: Spec, seed: Optional[int] = None, margin_check: bool = True) -> dict:
    """Draw one batch for `spec`. Deterministic in (spec, seed)."""
    if seed is None:
        seed = config_seed(spec.name)
    rng = np.random.default_rng(seed)
    n_max = _max_steps(spec)
    G, Rg, d = spec.groups, spec.rollouts, spec.d

    group_off = np.arange(G + 1, dtype=np.int32) * Rg
    steps_per_rollout, lens, store, planted, rewards = [], [], [], [], []
    resampled = 0
    for g in range(G):
        cents = _unit(rng, spec.centroids, d)
        if spec.rewards[0] == "bernoulli":
            p = spec.rewards[1]
        else:
            p = rng.beta(spec.rewards[1], spec.rewards[2])
        ns = [_n_steps(rng, spec) for _ in range(Rg)]
        for n in ns:
            lens.append(_lengths(rng, spec, n))
        steps_per_rollout.extend(ns)
        roll = np.repeat(np.arange(Rg), ns)
        depth = np.concatenate([np.arange(1, n + 1) for n in ns]) if Rg else np.zeros(0, dtype=np.int64)
        z, cid = _draw_states(rng, spec, cents, depth, n_max)
        s, e = _round(spec, z)
        rewards.extend((rng.random(Rg) < p).astype(np.uint8).tolist())
        if margin_check:
            resampled += _margin_filter(rng, spec, cents, n_max, s, e, cid, roll, depth)
        store.append(s)
        planted.append(cid)

    rollout_step_off = np.zeros(len(steps_per_rollout) + 1, dtype=np.int32)
    rollout_step_off[1:] = np.cumsum(steps_per_rollout)
    step_len = np.concatenate(lens).astype(np.int32) if lens else np.zeros(0, dtype=np.int32)
    rollout_token_off = np.zeros(len(steps_per_rollout) + 1, dtype=np.int64)
    if len(step_len):
        rollout_token_off[1:] = np.cumsum(np.add.reduceat(step_len.astype(np.int64), rollout_step_off[:-1]))
    emb = np.concatenate(store) if store else np.zeros((0, d))
    emb = emb.astype(np.uint16 if spec.dtype == "bf16" else np.float32)
    return dict(
        spec=spec,
        seed=seed,
        group_rollout_off=group_off,
        rollout_step_off=rollout_step_off,
        step_len=step_len,
        rollout_token_off=rollout_token_off,
        emb=np.ascontiguousarray(emb),
        emb_dtype=spec.dtype,
        reward=np.asarray(rewards, dtype=np.uint8),
        planted_centroid=np.concatenate(planted).astype(np.int32) if planted else np.zeros(0, np.int32),
        kappa=spec.kappa,
        w=spec.w,
        lambda_eff=spec.lambda_eff,
        margin_resampled=resampled,
    )


def _margin_filter(rng, spec, cents, n_max, store, exact, cid, roll, depth, comparable=None) -> int:
    """Redraw states whose cosine with a comparable state lies within `margin` of kappa
    (in place).  Comparable: another rollout (chain layout), or `comparable(rows)`, a
    [len(rows), n] boolean matrix."""
    redraws = 0
    rows = np.arange(len(exact))
    for _ in range(1000):
        nrm = np.linalg.norm(exact, axis=1)
        nrm[nrm == 0] = 1.0
        Zn = exact / nrm[:, None]
        C = Zn[rows] @ Zn.T
        bad = np.abs(C - spec.kappa) < spec.margin
        if comparable is None:
            bad &= roll[rows][:, None] != roll[None, :]
        else:
            bad &= comparable(rows)
        ii, jj = np.nonzero(bad)
        if len(ii) == 0:
            return redraws
        victims = np.unique(np.maximum(rows[ii], jj))
        z, c = _draw_states(rng, spec, cents, depth[victims], n_max)
        s, e = _round(spec, z)
        store[victims] = s
        exact[victims] = e
        cid[victims] = c
        redraws += len(victims)
        rows = victims
    raise RuntimeError("margin filter did not converge")


def _tree_shape(rng, spec: TreeSpec):
    """Parents (group-local, -1 = root) and depths of one group, in pre-order."""
    H = len(spec.schedule)
    par, dep = [], []

    def expand(p, h):  # children of node p (-1 = root) at depth h
        for _ in range(spec.schedule[h]):
            v = len(par)
            par.append(p)
            dep.append(h + 1)
            if h + 1 < H and not (rng.random() < spec.p_stop):
                expand(v, h + 1)

    expand(-1, 0)
    return np.asarray(par, dtype=np.int32), np.asarray(dep, dtype=np.int64)


def subtree_end(parent: np.ndarray) -> np.ndarray:
    """End (exclusive, group-local) of each state's subtree for a pre-order group."""
    n = len(parent)
    end = np.arange(1, n + 1, dtype=np.int64)
    for v in range(n - 1, -1, -1):
        if parent[v] >= 0:
            end[parent[v]] = max(end[parent[v]], end[v])
    return end


def make_tree_batch(spec: TreeSpec, seed: Optional[int] = None, margin_check: bool = True) -> dict:
    """Draw one tree-layout batch for `spec`.  Deterministic in (spec, seed)."""
    if seed is None:
        seed = config_seed(spec.name)
    rng = np.random.default_rng(seed)
    H, G, d = len(spec.schedule), spec.groups, spec.d
    n_band = max(H, spec.centroids // 2)  # depth span of the centroid bands
    pars, lens, store, planted, rewards, nleaf, nstate = [], [], [], [], [], [], []
    resampled = 0
    for g in range(G):
        cents = _unit(rng, spec.centroids, d)
        if spec.rewards[0] == "bernoulli":
            p = spec.rewards[1]
        else:
            p = rng.beta(spec.rewards[1], spec.rewards[2])
        par, dep = _tree_shape(rng, spec)
        n = len(par)
        end = subtree_end(par)
        leaves = int(np.sum(end == np.arange(1, n + 1)))
        lens.append(rng.integers(spec.lengths[1], spec.lengths[2] + 1, size=n).astype(np.int32))
        z, cid = _draw_states(rng, spec, cents, dep, n_band)
        s, e = _round(spec, z)
        rewards.extend((rng.random(leaves) < p).astype(np.uint8).tolist())
        if margin_check:
            idx = np.arange(n)

            def comparable(rows, end=end, idx=idx):
                r = rows[:, None]
                return ((idx[None, :] >= end[r]) | (r >= end[idx][None, :])) & (r != idx[None, :])

            resampled += _margin_filter(rng, spec, cents, n_band, s, e, cid, None, dep, comparable)
        pars.append(par)
        store.append(s)
        planted.append(cid)
        nleaf.append(leaves)
        nstate.append(n)
    step_len = np.concatenate(lens).astype(np.int32) if lens else np.zeros(0, np.int32)
    gso = np.zeros(G + 1, dtype=np.int32)
    gso[1:] = np.cumsum(nstate)
    gro = np.zeros(G + 1, dtype=np.int32)
    gro[1:] = np.cumsum(nleaf)
    gto = np.zeros(G + 1, dtype=np.int64)
    if len(step_len):
        gto[1:] = np.cumsum([int(l.astype(np.int64).sum()) for l in lens])
    emb = np.concatenate(store) if store else np.zeros((0, d))
    emb = emb.astype(np.uint16 if spec.dtype == "bf16" else np.float32)
    return dict(
        spec=spec, seed=seed, layout="tree",
        group_rollout_off=gro, group_state_off=gso,
        parent=np.concatenate(pars).astype(np.int32) if pars else np.zeros(0, np.int32),
        step_len=step_len, group_token_off=gto, total_tokens=int(gto[-1]),
        emb=np.ascontiguousarray(emb), emb_dtype=spec.dtype,
        reward=np.asarray(rewards, dtype=np.uint8),
        planted_centroid=np.concatenate(planted).astype(np.int32) if planted else np.zeros(0, np.int32),
        kappa=spec.kappa, w=spec.w, lambda_eff=spec.lambda_eff, margin_resampled=resampled,
    )


def is_tree(batch: dict) -> bool:
    return batch.get("parent") is not None


def as_tree(batch: dict) -> dict:
    """The same chain-layout batch written in the tree layout: each rollout is a path
    from the root, its last state its leaf; tokens stay where they are."""
    go, so, to = batch["group_rollout_off"], batch["rollout_step_off"], batch["rollout_token_off"]
    N = int(so[-1])
    gso = so[go].astype(np.int32)
    parent = np.arange(N, dtype=np.int64) - np.repeat(gso[:-1], np.diff(gso)) - 1
    first = so[:-1]
    parent[first] = -1
    out = {k: v for k, v in batch.items() if k not in ("rollout_step_off", "rollout_token_off")}
    out.update(layout="tree", group_state_off=gso, parent=parent.astype(np.int32),
               group_token_off=to[go].astype(np.int64), total_tokens=int(to[-1]))
    return out


def sub_batch(batch: dict, groups) -> dict:
    if is_tree(batch):
        return _sub_batch_tree(batch, groups)
    return _sub_batch_chain(batch, groups)


def _sub_batch_tree(batch: dict, groups) -> dict:
    groups = list(groups)
    go, gs, gt = batch["group_rollout_off"], batch["group_state_off"], batch["group_token_off"]
    rolls, states, toks = [], [], []
    ro, so, to = [0], [0], [0]
    for g in groups:
        rolls.append(np.arange(go[g], go[g + 1]))
        states.append(np.arange(gs[g], gs[g + 1]))
        toks.append((int(gt[g]), int(gt[g + 1])))
        ro.append(ro[-1] + int(go[g + 1] - go[g]))
        so.append(so[-1] + int(gs[g + 1] - gs[g]))
        to.append(to[-1] + int(gt[g + 1] - gt[g]))
    rolls = np.concatenate(rolls) if rolls else np.zeros(0, dtype=np.int64)
    states = np.concatenate(states) if states else np.zeros(0, dtype=np.int64)
    out = dict(batch)
    out.update(
        group_rollout_off=np.asarray(ro, dtype=np.int32), group_state_off=np.asarray(so, dtype=np.int32),
        group_token_off=np.asarray(to, dtype=np.int64), total_tokens=int(to[-1]),
        parent=batch["parent"][states].astype(np.int32), step_len=batch["step_len"][states].astype(np.int32),
        emb=np.ascontiguousarray(batch["emb"][states]), reward=batch["reward"][rolls].astype(np.uint8),
        planted_centroid=batch["planted_centroid"][states], source_groups=groups,
        source_rollouts=rolls, source_states=states, source_token_spans=toks,
    )
    return out


def _sub_batch_chain(batch: dict, groups) -> dict:
    """The batch restricted to the listed prompt groups (in the given order).

    Groups are independent in the method, so a sub-batch's outputs equal the
    corresponding slices of the full batch's outputs.
    """
    groups = list(groups)
    go, so, to = batch["group_rollout_off"], batch["rollout_step_off"], batch["rollout_token_off"]
    rolls, states, ro_n, steps = [], [], [0], [0]
    tok_spans = []
    for g in groups:
        r0, r1 = int(go[g]), int(go[g + 1])
        rolls.append(np.arange(r0, r1))
        s0, s1 = int(so[r0]), int(so[r1])
        states.append(np.arange(s0, s1))
        ro_n.append(ro_n[-1] + (r1 - r0))
    rolls = np.concatenate(rolls) if rolls else np.zeros(0, dtype=np.int64)
    states = np.concatenate(states) if states else np.zeros(0, dtype=np.int64)
    n_steps = (so[rolls + 1] - so[rolls]).astype(np.int64)
    rso = np.zeros(len(rolls) + 1, dtype=np.int32)
    rso[1:] = np.cumsum(n_steps)
    ntok = (to[rolls + 1] - to[rolls]).astype(np.int64)
    rto = np.zeros(len(rolls) + 1, dtype=np.int64)
    rto[1:] = np.cumsum(ntok)
    out = dict(batch)
    out.update(
        group_rollout_off=np.asarray(ro_n, dtype=np.int32),
        rollout_step_off=rso,
        step_len=batch["step_len"][states].astype(np.int32),
        rollout_token_off=rto,
        emb=np.ascontiguousarray(batch["emb"][states]),
        reward=batch["reward"][rolls].astype(np.uint8),
        planted_centroid=batch["planted_centroid"][states],
        source_groups=groups,
        source_rollouts=rolls,
        source_states=states,
    )
    return out


def token_index(batch: dict, sub: dict) -> np.ndarray:
    """For a sub-batch, the packed token positions of its tokens in the full batch."""
    if is_tree(sub):
        parts = [np.arange(a, b) for a, b in sub["source_token_spans"]]
        return np.concatenate(parts) if parts else np.zeros(0, dtype=np.int64)
    to = batch["rollout_token_off"]
    parts = [np.arange(to[r], to[r + 1]) for r in sub["source_rollouts"]]
    return np.concatenate(parts) if parts else np.zeros(0, dtype=np.int64)


def summary(batch: dict) -> dict:
    if is_tree(batch):
        go, gs = batch["group_rollout_off"], batch["group_state_off"]
        G = len(gs) - 1
        ng = np.diff(gs).astype(int).tolist()
        return dict(groups=G, rollouts=int(go[-1]), states=int(gs[-1]), tokens=int(batch["group_token_off"][-1]),
                    d=int(batch["emb"].shape[1]), dtype=batch["emb_dtype"], layout="tree",
                    max_states_per_group=max(ng) if ng else 0,
                    mean_states_per_group=(sum(ng) / G) if G else 0.0)
    go, so = batch["group_rollout_off"], batch["rollout_step_off"]
    G = len(go) - 1
    R = len(so) - 1
    N = int(so[-1])
    T = int(batch["rollout_token_off"][-1])
    ng = [int(so[go[g + 1]] - so[go[g]]) for g in range(G)]
    return dict(groups=G, rollouts=R, states=N, tokens=T, d=int(batch["emb"].shape[1]),
                dtype=batch["emb_dtype"], max_states_per_group=max(ng) if ng else 0,
                mean_states_per_group=(sum(ng) / G) if G else 0.0)


# ---- per-token log-probabilities for the policy loss (GraphPO Sec. 4.5) -------------
#
# Recipe (seed 20261202 + 100 + k by default): old log-probs -|N(0, 1.5)| - 0.01 (a
# sampled token's log-probability under the behaviour policy), new log-probs = old +
# N(0, 0.15) (a policy a few optimiser steps later: about a fifth of the tokens leave
# the clip range [0.8, 1.2]), reference log-probs = new + N(0, 0.1); all float32.
# Margin: tokens whose ratio exp(new - old) (fp64 on the float32 values) lies within
# 1e-4 of a clip bound are redrawn, so that the clip decision is unambiguous in fp32.
LOGP_SEED_OFFSET = 100


def make_logprobs(T: int, seed: int, clip_low: float = 0.2, clip_high: float = 0.2, margin: float = 1e-4,
                  spread: float = 0.15) -> dict:
    rng = np.random.default_rng(seed)
    old = (-np.abs(rng.normal(0.0, 1.5, T)) - 0.01).astype(np.float32)
    new = (old.astype(np.float64) + rng.normal(0.0, spread, T)).astype(np.float32)
    bounds = (1.0 - clip_low, 1.0 + clip_high)
    for _ in range(100):
        r = np.exp(new.astype(np.float64) - old.astype(np.float64))
        bad = np.zeros(T, dtype=bool)
        for c in bounds:
            bad |= np.abs(r - c) < margin
        if not bad.any():
            break
        new[bad] = (old[bad].astype(np.float64) + rng.normal(0.0, spread, int(bad.sum()))).astype(np.float32)
    else:
        raise RuntimeError("log-prob margin filter did not converge")
    ref = (new.astype(np.float64) + rng.normal(0.0, 0.1, T)).astype(np.float32)
    return dict(logp=new, old_logp=old, ref_logp=ref)


# ---- layer-by-layer views of a branching batch (per-layer merge, GraphPO Sec. 4.2) -----


def tree_depths(batch: dict) -> np.ndarray:
    """Depth of every state of a tree-layout batch (1 = child of the prompt root)."""
    par, gs = batch["parent"], batch["group_state_off"]
    dep = np.zeros(len(par), dtype=np.int64)
    for g in range(len(gs) - 1):
        s0 = int(gs[g])
        for v in range(s0, int(gs[g + 1])):
            dep[v] = 1 if par[v] < 0 else dep[s0 + par[v]] + 1
    return dep


def truncate_tree(batch: dict, layer: int) -> dict:
    """The batch as it stands after layer `layer` is sampled: the states of depth <= layer
    (pre-order is kept, parents renumbered), their edges' tokens, the leaves of that tree
    as its rollouts with placeholder rewards 0 (no answer is verified yet), and `active`:
    1 on the states of depth `layer` that the full batch expands further."""
    par, gs = batch["parent"], batch["group_state_off"]
    dep = tree_depths(batch)
    has_child = np.zeros(len(par), dtype=bool)
    for g in range(len(gs) - 1):
        s0 = int(gs[g])
        for v in range(s0, int(gs[g + 1])):
            if par[v] >= 0:
                has_child[s0 + par[v]] = True
    keep = dep <= layer
    new_par, new_gs, new_go, new_gt, leaves = [], [0], [0], [0], 0
    for g in range(len(gs) - 1):
        s0, s1 = int(gs[g]), int(gs[g + 1])
        idx = np.nonzero(keep[s0:s1])[0]
        local = -np.ones(s1 - s0, dtype=np.int64)
        local[idx] = np.arange(len(idx))
        p = par[s0:s1][idx]
        new_par.append(np.where(p < 0, -1, local[np.maximum(p, 0)]).astype(np.int32))
        child = np.zeros(len(idx), dtype=bool)
        q = new_par[-1]
        child[q[q >= 0]] = True
        nl = int((~child).sum())
        leaves += nl
        new_gs.append(new_gs[-1] + len(idx))
        new_go.append(new_go[-1] + nl)
        new_gt.append(new_gt[-1] + int(batch["step_len"][s0:s1][idx].astype(np.int64).sum()))
    states = np.nonzero(keep)[0]
    out = {k: v for k, v in batch.items() if k not in ("planted_centroid",)}
    out.update(parent=np.concatenate(new_par) if new_par else np.zeros(0, np.int32),
               group_state_off=np.asarray(new_gs, np.int32), group_rollout_off=np.asarray(new_go, np.int32),
               group_token_off=np.asarray(new_gt, np.int64), total_tokens=int(new_gt[-1]),
               step_len=batch["step_len"][states].astype(np.int32), emb=np.ascontiguousarray(batch["emb"][states]),
               reward=np.zeros(leaves, np.uint8), source_states=states,
               active=((dep[states] == layer) & has_child[states]).astype(np.uint8), layer=layer)
    return out
