"""GraphPO policy loss on per-token log-probabilities -- CPU ORACLE.

Test infrastructure only: the tests, `__graft_entry__.smoke()` and the
benchmark's CPU-baseline leg use it; the product path never imports it.
Plain numpy in fp64, one formula per line, following

  Sec. 4.5 (objective J_GraphPO, built on DAPO's clipped surrogate):
      J = E_q [ 1/|E| sum_{e in E} 1/|e| sum_{t=1}^{|e|}
                ( min(r_t A(e), clip(r_t, 1 - eps, 1 + eps) A(e)) - beta D_KL ) ],
      r_t = pi_theta(o_t | .) / pi_old(o_t | .), E = the direct edges of a prompt's
      graph, |e| = tokens of edge e, every token of an edge with the edge's A_dual;
  Algorithm S.1, Stage 4 (the split form):
      L_ppo(A_cor, m_resp) + lambda_eff L_ppo(A_eff, m_eff) + beta L_KL.

Readings (the paper leaves these open):
  * E_q over a batch = the mean over its prompt groups that have edges; "edge"
    normalisation.  "token" normalisation is DAPO's token mean 1/T sum_t.
  * the clip range is [1 - clip_low, 1 + clip_high] (the paper's symmetric
    0.2 by default; DAPO decouples the two bounds);
  * D_KL per token is the k3 estimate exp(x) - x - 1, x = log pi_ref - log pi_theta
    (non-negative, unbiased for KL(pi_theta || pi_ref) under pi_theta);
  * split form: each term is the surrogate above with its own advantage; the mask
    multiplies the token terms and leaves the normalisation alone (m_resp = 1 on
    every generated token);
  * the loss is L = -J; its derivative with respect to log pi_theta of a token
    is taken where the min picks the unclipped term (r A <= clip(r) A, which
    includes every ratio inside the clip range): there d(r A)/d log pi = r A,
    elsewhere the surrogate is constant; the entropy bonus of Algorithm S.1 needs
    the whole vocabulary distribution and is not part of a token-level loss.
"""
from __future__ import annotations

import numpy as np


def edge_of_token(batch: dict):
    """Edge (state) index of every token and the token's edge length |e|, from the
    batch layout: chain layout -- rollout r's tokens start at rollout_token_off[r]
    and hold its steps in order; tree layout -- group g's tokens start at
    group_token_off[g] and hold its states' edges in state order."""
    sl = np.asarray(batch["step_len"], dtype=np.int64)
    T = int(batch["group_token_off"][-1] if batch.get("parent") is not None else batch["rollout_token_off"][-1])
    edge = np.full(T, -1, dtype=np.int64)
    if batch.get("parent") is not None:
        spans = [(int(batch["group_token_off"][g]), int(batch["group_state_off"][g]), int(batch["group_state_off"][g + 1]))
                 for g in range(len(batch["group_state_off"]) - 1)]
    else:
        so, to = batch["rollout_step_off"], batch["rollout_token_off"]
        spans = [(int(to[r]), int(so[r]), int(so[r + 1])) for r in range(len(so) - 1)]
    for t0, v0, v1 in spans:
        t = t0
        for v in range(v0, v1):
            edge[t:t + sl[v]] = v
            t += sl[v]
    assert (edge >= 0).all(), "token spans do not tile the tokens"
    return edge, sl[edge]


def group_of_state(batch: dict) -> np.ndarray:
    N = len(batch["step_len"])
    grp = np.empty(N, dtype=np.int64)
    go = batch["group_rollout_off"]
    for g in range(len(go) - 1):
        if batch.get("parent") is not None:
            a, b = batch["group_state_off"][g], batch["group_state_off"][g + 1]
        else:
            a, b = batch["rollout_step_off"][go[g]], batch["rollout_step_off"][go[g + 1]]
        grp[a:b] = g
    return grp


def token_weights(batch: dict, norm: str = "edge") -> np.ndarray:
    """Weight of every token in J: "edge" -- 1 / (G' |E_g| |e|) with G' the groups
    that have edges and |E_g| = the group's direct edges (one per state); "token" -- 1/T."""
    edge, elen = edge_of_token(batch)
    T = len(edge)
    if norm == "token":
        return np.full(T, 1.0 / T if T else 0.0)
    grp = group_of_state(batch)
    G = len(batch["group_rollout_off"]) - 1
    n_edges = np.bincount(grp, minlength=G).astype(np.float64)  # |E_g|
    G_nonempty = float(np.count_nonzero(n_edges))
    return 1.0 / (G_nonempty * n_edges[grp[edge]] * elen.astype(np.float64))


def surrogate(ratio: np.ndarray, A: np.ndarray, clip_low: float, clip_high: float):
    """min(r A, clip(r, 1 - clip_low, 1 + clip_high) A), its derivative with respect to
    log r (r A where the unclipped term is the minimum, else 0) and whether the clipped
    term was strictly smaller."""
    unclipped = ratio * A
    clipped = np.clip(ratio, 1.0 - clip_low, 1.0 + clip_high) * A
    value = np.minimum(unclipped, clipped)
    takes_unclipped = unclipped <= clipped
    return value, np.where(takes_unclipped, ratio * A, 0.0), ~takes_unclipped


def kl_k3(x: np.ndarray):
    """The k3 estimate e^x - x - 1 (x = log pi_ref - log pi_theta) and its derivative with
    respect to log pi_theta, 1 - e^x."""
    return np.expm1(x) - x, -np.expm1(x)


def token_loss(batch: dict, logp, old_logp, ref_logp=None, edge_adv=None, edge_cor=None, edge_eff=None,
               edge_mask=None, clip_low: float = 0.2, clip_high: float = 0.2, beta: float = 0.0,
               lambda_eff: float = 1.0, form: str = "dual", norm: str = "edge") -> dict:
    """L = -J on one batch.  Returns loss, grad (dL/dlogp per token), the policy term
    J_pg = sum_t w_t (surrogate), the KL term sum_t w_t k3_t, the number of tokens whose
    (first) surrogate was clipped and the token mean of the ratio."""
    edge, _ = edge_of_token(batch)
    w = token_weights(batch, norm)
    logp = np.asarray(logp, dtype=np.float64)
    old = np.asarray(old_logp, dtype=np.float64)
    ratio = np.exp(logp - old)
    if form == "dual":
        f, df, clipped = surrogate(ratio, np.asarray(edge_adv, dtype=np.float64)[edge], clip_low, clip_high)
    elif form == "split":
        f1, df1, clipped = surrogate(ratio, np.asarray(edge_cor, dtype=np.float64)[edge], clip_low, clip_high)
        f2, df2, _ = surrogate(ratio, np.asarray(edge_eff, dtype=np.float64)[edge], clip_low, clip_high)
        m = np.asarray(edge_mask, dtype=np.float64)[edge]
        f = f1 + lambda_eff * m * f2
        df = df1 + lambda_eff * m * df2
    else:
        raise ValueError(form)
    if beta != 0.0:
        kl, dkl = kl_k3(np.asarray(ref_logp, dtype=np.float64) - logp)
    else:
        kl = dkl = np.zeros_like(logp)
    j_pg = float(np.sum(w * f))
    j_kl = float(np.sum(w * kl))
    loss = -(j_pg - beta * j_kl)
    grad = -w * df + beta * w * dkl
    T = len(edge)
    return dict(loss=loss, grad=grad, pg=j_pg, kl=j_kl, clipped=int(np.count_nonzero(clipped)),
                ratio_mean=float(ratio.mean()) if T else 0.0, weights=w)
