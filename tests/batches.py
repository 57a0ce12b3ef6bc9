"""Small hand-built batches for tests (chain layout, see workloads.py)."""
import numpy as np


def from_rollouts(groups, d=None, dtype="f32", kappa=0.9, w=0.7, lambda_eff=1.0, root_emb=None):
    """groups: list of groups; a group is a list of rollouts (emb_rows, step_lens, reward)."""
    go, so, sl, emb, rew = [0], [0], [], [], []
    for grp in groups:
        for rows, lens, r in grp:
            assert len(rows) == len(lens) and len(rows) >= 1
            emb.extend(rows)
            sl.extend(lens)
            so.append(so[-1] + len(rows))
            rew.append(r)
        go.append(len(rew))
    emb = np.asarray(emb, dtype=np.float64)
    if d is None:
        d = emb.shape[1]
    sl = np.asarray(sl, dtype=np.int32)
    so = np.asarray(so, dtype=np.int32)
    to = np.zeros(len(so), dtype=np.int64)
    for r in range(len(so) - 1):
        to[r + 1] = to[r] + int(sl[so[r]:so[r + 1]].sum())
    if dtype == "bf16":
        from paper_2606_18954_gb300.workloads import f32_to_bf16_bits
        e = f32_to_bf16_bits(emb.astype(np.float32))
        root = f32_to_bf16_bits(np.asarray(root_emb, np.float32)) if root_emb is not None else None
    else:
        e = emb.astype(np.float32)
        root = np.asarray(root_emb, np.float32) if root_emb is not None else None
    b = dict(group_rollout_off=np.asarray(go, np.int32), rollout_step_off=so, step_len=sl,
             rollout_token_off=to, emb=e, emb_dtype=dtype, reward=np.asarray(rew, np.uint8),
             kappa=kappa, w=w, lambda_eff=lambda_eff)
    if root is not None:
        b["root_emb"] = root
    return b


def states_of(batch):
    """(rollout, depth, group) of every state."""
    go, so = batch["group_rollout_off"], batch["rollout_step_off"]
    R = len(so) - 1
    roll = np.repeat(np.arange(R), np.diff(so))
    depth = np.concatenate([np.arange(1, n + 1) for n in np.diff(so)]) if R else np.zeros(0, int)
    grp_of_roll = np.repeat(np.arange(len(go) - 1), np.diff(go))
    return roll, depth, grp_of_roll[roll] if R else np.zeros(0, int)


def emb_f64(batch):
    e = batch["emb"]
    if batch["emb_dtype"] == "bf16":
        return (e.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return e.astype(np.float64)
