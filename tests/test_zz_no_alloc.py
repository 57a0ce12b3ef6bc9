"""gpo_compute_noalloc, the allocation-free entry point, against gpo_compute.

Some callers cannot allocate device memory when they need the advantages (a
trainer whose memory is all owned by a framework pool, a plug-in whose host
forbids allocation calls, a loop that cannot take cudaMalloc's implicit
synchronisation); gpo_compute_noalloc serves them from one scratch array built
into the library.  These tests call it through the C ABI twice in a row, on
different batches (the scratch keeps the previous call's contents, which must
not leak into the next result): chain batches on the group-resident path, a
tree-layout batch, fp32 embeddings (CUDA-core path) and a batch on the tiled
path whose workspace nearly fills the scratch.  Every output is compared with
gpo_compute's within the parity tolerance (class ids exactly).  A second call
must leave the device's free memory unchanged (nothing allocated), and a batch
one workspace step above the scratch is refused before anything is enqueued.
This file is collected last and also passes on its own in a fresh process.
"""
import ctypes

import numpy as np
import pytest

from paper_2606_18954_gb300 import workloads as W

pytestmark = pytest.mark.gpu

RTOL, ATOL = 1e-5, 1e-6
KEYS = ("adv", "adv_cor", "adv_eff", "eff_mask", "class_id", "node_score", "edge_adv", "edge_cor", "edge_eff",
        "edge_eff_mask", "group_eff", "group_eff_graph")  # the order of gpo_outputs
SCRATCH = 32 << 20  # GPO_NOALLOC_SCRATCH_BYTES


@pytest.fixture(scope="module")
def P():
    import torch
    if not torch.cuda.is_available():
        pytest.fail("a CUDA device is required for -m gpu tests")
    import paper_2606_18954_gb300 as pkg
    pkg.build()
    return pkg


def _noalloc(P, gp, cb, out):
    import torch
    B = P.binding
    co = B.COutputs(*[out[k].data_ptr() if out.get(k) is not None and out[k].numel() else None for k in KEYS])
    stream = torch.cuda.current_stream()
    return P.load().gpo_compute_noalloc(gp._h, ctypes.byref(cb), ctypes.byref(co), ctypes.c_void_p(stream.cuda_stream))


def _assert_same(got, ref):
    for k in KEYS:
        if k not in ref:
            continue
        g, r = got[k].cpu().numpy(), ref[k].cpu().numpy()
        if g.dtype.kind in "iu":
            np.testing.assert_array_equal(g, r, err_msg=k)
        else:
            err = np.abs(g.astype(np.float64) - r.astype(np.float64))
            assert np.all(err <= RTOL * np.abs(r.astype(np.float64)) + ATOL), (k, float(err.max()))


def _check(P, b, maxn=None, all_outputs=True):
    """gpo_compute_noalloc twice on the batch (the second call with the memory check)
    against gpo_compute."""
    import torch
    gp = P.GraphPO(kappa=b["kappa"], w=b["w"], lambda_eff=b["lambda_eff"])
    db = P.Batch.from_arrays(b, device="cuda")
    cb = db.c_struct()
    if maxn is not None:
        cb.max_states_per_group = maxn
    kw = dict(components=True, nodes=True, edges=True, efficiency=True) if all_outputs else {}
    ref = gp.alloc_outputs(db, **kw)
    ws = torch.empty(P.binding.workspace_size(cb, gp._h), dtype=torch.uint8, device="cuda")
    co = P.binding._c_outputs(ref)
    code = P.load().gpo_compute(gp._h, ctypes.byref(cb), ctypes.byref(co), ws.data_ptr(), ws.numel(),
                                ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert code == 0, gp.last_error()
    gp.check()
    for call in range(2):
        out = gp.alloc_outputs(db, **kw)
        for o in out.values():
            o.fill_(7) if o.dtype != torch.float32 else o.fill_(float("nan"))
        torch.cuda.synchronize()
        free0 = torch.cuda.mem_get_info()[0]
        assert _noalloc(P, gp, cb, out) == 0, gp.last_error()
        gp.check()
        torch.cuda.synchronize()
        if call == 1:  # the first call may load kernels; the second allocates nothing
            assert torch.cuda.mem_get_info()[0] == free0
        _assert_same(out, ref)
    return gp, db, cb


def test_noalloc_matches_compute_twice(P):
    for name, groups in (("math", 4), ("agentic", 12)):
        _check(P, W.make_batch(W.CONFIGS[name].scaled(groups)))


def test_noalloc_tree_layout_and_fp32(P):
    _check(P, W.make_tree_batch(W.TREE_CONFIGS["tree"].scaled(groups=6)))
    _check(P, W.make_batch(W.CONFIGS["tiny"]))


def test_noalloc_near_the_scratch_size(P):
    """A batch whose workspace is the largest one of its shape that fits the scratch
    (max_states_per_group raised, which sizes the workspace and selects the tiled path) runs
    and matches gpo_compute; the same batch one workspace step above is refused."""
    b = W.make_batch(W.CONFIGS["full"].scaled(groups=256), margin_check=False)
    gp = P.GraphPO(kappa=b["kappa"], w=b["w"], lambda_eff=b["lambda_eff"])
    cb = P.Batch.from_arrays(b, device="cpu").c_struct()
    size = lambda m: (setattr(cb, "max_states_per_group", m), P.binding.workspace_size(cb))[1]
    lo, hi = int(cb.max_states_per_group), 4096
    assert size(lo) <= SCRATCH < size(hi)
    while hi - lo > 1:  # largest max_states_per_group whose workspace fits
        mid = (lo + hi) // 2
        lo, hi = (mid, hi) if size(mid) <= SCRATCH else (lo, mid)
    assert size(lo) <= SCRATCH < size(hi)
    _check(P, b, maxn=lo, all_outputs=False)
    import torch
    db = P.Batch.from_arrays(b, device="cuda")
    cbd = db.c_struct()
    cbd.max_states_per_group = hi
    out = gp.alloc_outputs(db)
    assert _noalloc(P, gp, cbd, out) == 8
    assert "built-in scratch" in gp.last_error()
    torch.cuda.synchronize()


def test_noalloc_rejects_batches_above_its_scratch(P):
    """A batch whose workspace exceeds GPO_NOALLOC_SCRATCH_BYTES is refused before any
    launch (only host-side sizes are read; nothing is dereferenced)."""
    b = W.make_batch(W.CONFIGS["math"].scaled(2))
    gp = P.GraphPO(kappa=b["kappa"], w=b["w"], lambda_eff=b["lambda_eff"])
    db = P.Batch.from_arrays(b, device="cuda")
    out = gp.alloc_outputs(db)
    cb = db.c_struct()
    cb.num_states = 1 << 24
    cb.max_states_per_group = 4096
    import torch
    code = _noalloc(P, gp, cb, out)
    assert code == 8, code
    assert "built-in scratch" in gp.last_error()
    cb.num_states = -1  # a host-checkable error: the message is this call's, not the last one's
    assert _noalloc(P, gp, cb, out) == 1
    assert "negative" in gp.last_error()
