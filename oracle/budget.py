"""Per-layer merge and next-layer budgets of GraphPO's graph construction -- CPU ORACLE.

Test infrastructure only: the tests, `__graft_entry__.smoke()` and the benchmark's
CPU-baseline leg use it; the product path never imports it.

GraphPO grows the graph layer by layer (Algorithm S.1, Stage 1): after the states of
layer h are registered, every non-causal pair is tested and linked (Sec. 4.2), and a
path that reaches an existing equivalence class has its next-layer budget halved,
keeping at least one continuation; the saved budget goes to the active frontier states
that are not redundant (Sec. 4.2, and the budget-reallocation proposition).  This
oracle follows those steps on the batch as it stands after layer h (states of depth
<= h, a tree-layout batch):

  * classes: the C oracle's equivalence classes of that batch (all non-causal pairs of
    states of depth <= h; the pairs of earlier layers were linked by earlier calls, so
    the union is the same);
  * the frontier: states of depth h that are active (to be expanded);
  * a frontier state v is redundant when its class holds a state registered before v:
    one of an earlier layer, or one of layer h that precedes v (states of a layer are
    registered in index order);
  * budget b_v = b_next for a non-redundant frontier state, max(1, floor(b_next / 2))
    for a redundant one, 0 off the frontier;
  * the saved budget S = sum over redundant frontier states of (b_next - their budget)
    is spread over the k non-redundant frontier states: floor(S / k) each, and one
    more to the first S mod k of them in registration order (with k = 0 it is not spent).

Readings (the paper leaves these open): "registered before" within a layer is index
order; the reallocation is the even split above; inactive frontier states (branches that
end) get no budget and take no share.
"""
from __future__ import annotations

import numpy as np


def depths(batch: dict) -> np.ndarray:
    par, gs = batch["parent"], batch["group_state_off"]
    dep = np.zeros(len(par), dtype=np.int64)
    for g in range(len(gs) - 1):
        s0 = int(gs[g])
        for v in range(s0, int(gs[g + 1])):
            dep[v] = 1 if par[v] < 0 else dep[s0 + par[v]] + 1
    return dep


def registered_before(dep, u: int, v: int) -> bool:
    """State u was registered before state v: an earlier layer, or the same layer and a
    smaller index."""
    return dep[u] < dep[v] or (dep[u] == dep[v] and u < v)


def halved(b_next: int) -> int:
    """The budget of a path that reached an existing class: half, at least one."""
    return max(1, b_next // 2)


def spread(saved: int, k: int):
    """The saved budget over k non-redundant states, in registration order: an even
    share each and one more for the first saved mod k."""
    share, extra = divmod(saved, k)
    return [share + (1 if rank < extra else 0) for rank in range(k)]


def layer_budget(batch: dict, layer: int, b_next: int, active=None, params: dict | None = None) -> dict:
    import oracle
    if batch.get("parent") is None:
        raise ValueError("the per-layer budget needs the tree layout")
    p = dict(params or {})
    out = oracle.run(batch, p, want=["class_id"])
    label = out["class_id"]
    dep = depths(batch)
    N = len(dep)
    act = np.ones(N, dtype=bool) if active is None else np.asarray(active).astype(bool)
    frontier = (dep == layer) & act
    half = halved(b_next)
    budget = np.zeros(N, dtype=np.int64)
    redundant = np.zeros(N, dtype=bool)
    gs = batch["group_state_off"]
    for g in range(len(gs) - 1):
        s0, s1 = int(gs[g]), int(gs[g + 1])
        saved, keep = 0, []
        for v in range(s0, s1):
            if not frontier[v]:
                continue
            for u in range(s0, s1):  # an earlier-registered member of v's class?
                if u != v and label[u] == label[v] and registered_before(dep, u, v):
                    redundant[v] = True
                    break
            if redundant[v]:
                budget[v] = half
                saved += b_next - half
            else:
                budget[v] = b_next
                keep.append(v)
        if keep:
            for v, more in zip(keep, spread(saved, len(keep))):
                budget[v] += more
    return dict(class_id=label, budget=budget, redundant=redundant, frontier=frontier)
