"""The bounded waits' failure path, run on purpose on the GPU.

Every mbarrier and flag wait in the tensor-core kernels gives up after a time limit, reports
GPO_ERR_TIMEOUT and lets the kernel wind down (copies in flight land, issued MMAs complete,
TMEM is released) instead of hanging.  GPO_FLAG_DEBUG_TIMEOUT makes the MMA warp's first wait
in every CTA run out (about a millisecond on an mbarrier nothing arrives on), so that this
path runs without any fault: each test checks that gpo_sync_status returns GPO_ERR_TIMEOUT,
twice in a row, and that the same CUDA context then computes the batch correctly (class ids
exactly, advantages within the parity bar, against the oracle).  Paths covered: the
group-resident kernel (both instances, chain and tree layouts) and the tiled tensor-core path.
"""
import numpy as np
import pytest

from paper_2606_18954_gb300 import workloads as W

pytestmark = pytest.mark.gpu

RTOL, ATOL = 1e-5, 1e-6
TIMEOUT = 7


@pytest.fixture(scope="module")
def P():
    import torch
    if not torch.cuda.is_available():
        pytest.fail("a CUDA device is required for -m gpu tests")
    import paper_2606_18954_gb300 as pkg
    pkg.build()
    return pkg


def _params(b):
    return dict(kappa=float(b["kappa"]), w=float(b["w"]), lambda_eff=float(b["lambda_eff"]), std_eps=1e-6,
                std_ddof=1, merge_rule=0)


def _close(got, ref64, name):
    ref = np.asarray(ref64, np.float64).astype(np.float32).astype(np.float64)
    err = np.abs(np.asarray(got, np.float64) - ref)
    assert np.all(err <= RTOL * np.abs(ref) + ATOL), (name, float(err.max()))


CASES = {
    "fused chain (384-state instance)": (lambda: W.make_batch(W.CONFIGS["math"].scaled(6)), 0),
    "fused chain (128-state instance)": (lambda: W.make_batch(W.CONFIGS["agentic"].scaled(12)), 0),
    "fused tree": (lambda: W.make_tree_batch(W.TREE_CONFIGS["tree"].scaled(groups=4)), 0),
    "tiled chain": (lambda: W.make_batch(W.CONFIGS["math"].scaled(6)), 2),
    "tiled tree": (lambda: W.make_tree_batch(W.TREE_CONFIGS["tree"].scaled(groups=4)), 2),
}


@pytest.mark.parametrize("case", list(CASES))
def test_forced_timeout_then_a_normal_call(P, case):
    import torch

    import oracle
    make, flags = CASES[case]
    b = make()
    p = _params(b)
    db = P.Batch.from_arrays(b, device="cuda")
    forced = P.GraphPO(kappa=p["kappa"], w=p["w"], lambda_eff=p["lambda_eff"],
                       flags=flags | P.binding.FLAG_DEBUG_TIMEOUT)
    out = forced.alloc_outputs(db)
    for _ in range(2):  # twice in a row on the same context and workspace
        forced.compute_into(db, out)
        with pytest.raises(P.GraphPOError) as e:
            forced.check()
        assert e.value.code == TIMEOUT, (case, e.value.code, forced.last_error())
    # the context is usable: the same batch, computed normally, matches the oracle
    gp = P.GraphPO(kappa=p["kappa"], w=p["w"], lambda_eff=p["lambda_eff"], flags=flags)
    res = gp(db, nodes=True)
    gp.check()
    torch.cuda.synchronize()
    got = {k: v.cpu().numpy() for k, v in res.items()}
    ref = oracle.run(b, p, threads=8)
    np.testing.assert_array_equal(got["class_id"], ref["class_id"], err_msg=case)
    _close(got["edge_adv"], ref["edge_adv"], f"{case} edge_adv")
    _close(got["adv"], ref["adv"], f"{case} adv")
    # and torch's own kernels still run on it
    x = torch.arange(1 << 20, device="cuda", dtype=torch.float32)
    assert float(x.sum().item()) == pytest.approx((1 << 20) * ((1 << 20) - 1) / 2, rel=1e-6)
