"""Per-layer graph construction on the GPU (gpo_layer_budget: classes of the states
sampled so far and next-layer budgets, GraphPO Sec. 4.2 and Algorithm S.1 Stage 1),
through the C ABI, against the CPU oracle: budgets and class ids bit-exact, layer by
layer, on the three similarity paths; after the last layer the classes equal gpo_compute's
on the whole batch."""
import functools

import numpy as np
import pytest

from oracle import budget as OB
from paper_2606_18954_gb300 import workloads as W
from test_gpu_parity import PATH_FLAGS, gp_mod, torch_cuda  # noqa: F401

pytestmark = pytest.mark.gpu

SPECS = {
    "sched25422": W.TreeSpec("sched25422", 4, (2, 5, 4, 2, 2), 64, "bf16", 8, 0.05, 0.9, ("per_step", 4, 64),
                             ("bernoulli", 0.5)),
    "sched4532": W.TreeSpec("sched4532", 3, (4, 5, 3, 2), 64, "bf16", 8, 0.05, 0.9, ("per_step", 8, 96),
                            ("bernoulli", 0.5)),
    "sched76543": W.TreeSpec("sched76543", 1, (7, 6, 5, 4, 3), 64, "bf16", 16, 0.05, 0.9, ("per_step", 4, 40),
                             ("bernoulli", 0.5)),
    "small_f32": W.TreeSpec("small_f32", 6, (2, 3, 3), 32, "f32", 6, 0.05, 0.9, ("per_step", 1, 9),
                            ("bernoulli", 0.5), p_stop=0.2),
}


@functools.lru_cache(maxsize=None)
def tree(name):
    return W.make_tree_batch(SPECS[name], seed=W.BASE_SEED + 400 + sorted(SPECS).index(name))


def run(P, t, layer, b_next, flags=0, active=True, kappa=0.9):
    import torch
    gp = P.GraphPO(kappa=kappa, flags=flags)
    db = P.Batch.from_arrays(t, device="cuda")
    act = torch.as_tensor(t["active"], device="cuda") if active else None
    out = gp.layer_budget(db, layer, b_next, act, classes=True)
    gp.check()
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in out.items()}


CASES = [("sched25422", "fused"), ("sched25422", "tiled"), ("sched4532", "fused"), ("sched4532", "simt"),
         ("sched76543", "tiled"), ("small_f32", "simt")]


@pytest.mark.parametrize("name,path", CASES)
@pytest.mark.parametrize("b_next", [1, 2, 5])
def test_layer_budgets(gp_mod, name, path, b_next):
    b = tree(name)
    if path != "simt" and b["emb_dtype"] != "bf16":
        pytest.skip("fp32 embeddings always use the CUDA-core similarity kernel")
    H = len(SPECS[name].schedule)
    seen_redundant = False
    for h in range(1, H + 1):
        t = W.truncate_tree(b, h)
        ref = OB.layer_budget(t, h, b_next, t["active"], dict(kappa=0.9))
        got = run(gp_mod, t, h, b_next, PATH_FLAGS[path])
        np.testing.assert_array_equal(got["class_id"], ref["class_id"], err_msg=f"{name} layer {h}")
        np.testing.assert_array_equal(got["budget"], ref["budget"], err_msg=f"{name} layer {h}")
        seen_redundant |= bool(ref["redundant"].any())
    assert seen_redundant


def test_all_frontier_active_and_final_layer_classes(gp_mod):
    """active = NULL: every state of the layer is on the frontier; after the last layer the
    classes are gpo_compute's on the whole batch."""
    import torch
    P = gp_mod
    b = tree("sched25422")
    H = len(SPECS["sched25422"].schedule)
    t = W.truncate_tree(b, 3)
    ref = OB.layer_budget(t, 3, 4, None, dict(kappa=0.9))
    got = run(P, t, 3, 4, active=False)
    np.testing.assert_array_equal(got["budget"], ref["budget"])
    last = run(P, W.truncate_tree(b, H), H, 2)
    gp = P.GraphPO(kappa=0.9)
    out = gp(P.Batch.from_arrays(b, device="cuda"), nodes=True)
    gp.check()
    np.testing.assert_array_equal(last["class_id"], out["class_id"].cpu().numpy())


def test_tree_workload_layer(gp_mod):
    """The full-size tree workload after layer 4 of 5 (the shape the benchmark times)."""
    b = W.make_tree_batch(W.TREE_CONFIGS["tree"])
    t = W.truncate_tree(b, 4)
    ref = OB.layer_budget(t, 4, 2, t["active"], dict(kappa=float(b["kappa"])))
    got = run(gp_mod, t, 4, 2, kappa=float(b["kappa"]))
    np.testing.assert_array_equal(got["class_id"], ref["class_id"])
    np.testing.assert_array_equal(got["budget"], ref["budget"])


def test_layer_budget_errors(gp_mod):
    import torch
    P = gp_mod
    gp = P.GraphPO(kappa=0.9)
    t = W.truncate_tree(tree("sched4532"), 2)
    db = P.Batch.from_arrays(t, device="cuda")
    for layer, b_next in ((0, 2), (2, 0), (2, 1 << 17)):
        with pytest.raises(P.GraphPOError) as e:
            gp.layer_budget(db, layer, b_next)
        assert e.value.code == 1
    chain = P.Batch.from_arrays(W.make_batch(W.CONFIGS["tiny"].scaled(2)), device="cuda")
    with pytest.raises(P.GraphPOError) as e:
        gp.layer_budget(chain, 2, 2)
    assert e.value.code == 5
