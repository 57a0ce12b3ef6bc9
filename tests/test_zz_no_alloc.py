"""gpo_compute_noalloc, the allocation-free entry point, against gpo_compute.

Some callers cannot allocate device memory when they need the advantages (a
trainer whose memory is all owned by a framework pool, a plug-in whose host
forbids allocation calls, a loop that cannot take cudaMalloc's implicit
synchronisation); gpo_compute_noalloc serves them from one scratch array built
into the library.  These tests call it through the C ABI twice in a row, on two
different batches (the scratch keeps the previous call's contents, which must
not leak into the next result), and compare every output with gpo_compute's
within the parity tolerance (class ids exactly).  This file is collected last
and also passes on its own in a fresh process.
"""
import ctypes

import numpy as np
import pytest

from paper_2606_18954_gb300 import workloads as W

pytestmark = pytest.mark.gpu

RTOL, ATOL = 1e-5, 1e-6
KEYS = ("adv", "adv_cor", "adv_eff", "eff_mask", "class_id", "node_score", "edge_adv", "edge_cor", "edge_eff",
        "edge_eff_mask", "group_eff", "group_eff_graph")  # the order of gpo_outputs


@pytest.fixture(scope="module")
def P():
    import torch
    if not torch.cuda.is_available():
        pytest.fail("a CUDA device is required for -m gpu tests")
    import paper_2606_18954_gb300 as pkg
    pkg.build()
    return pkg


def _noalloc(P, gp, db, out):
    import torch
    B = P.binding
    co = B.COutputs(*[out[k].data_ptr() if out.get(k) is not None and out[k].numel() else None for k in KEYS])
    cb = db.c_struct()
    stream = torch.cuda.current_stream()
    return P.load().gpo_compute_noalloc(gp._h, ctypes.byref(cb), ctypes.byref(co), ctypes.c_void_p(stream.cuda_stream))


def _assert_same(got, ref):
    for k in KEYS:
        g, r = got[k].cpu().numpy(), ref[k].cpu().numpy()
        if g.dtype.kind in "iu":
            np.testing.assert_array_equal(g, r, err_msg=k)
        else:
            err = np.abs(g.astype(np.float64) - r.astype(np.float64))
            assert np.all(err <= RTOL * np.abs(r.astype(np.float64)) + ATOL), (k, float(err.max()))


def test_noalloc_matches_compute_twice(P):
    import torch
    for name, groups in (("math", 4), ("agentic", 12)):
        b = W.make_batch(W.CONFIGS[name].scaled(groups))
        gp = P.GraphPO(kappa=b["kappa"], w=b["w"], lambda_eff=b["lambda_eff"])
        db = P.Batch.from_arrays(b, device="cuda")
        ref = gp(db, components=True, nodes=True, edges=True, efficiency=True)
        gp.check()
        out = gp.alloc_outputs(db, components=True, nodes=True, edges=True, efficiency=True)
        for o in out.values():
            o.fill_(7) if o.dtype != torch.float32 else o.fill_(float("nan"))
        assert _noalloc(P, gp, db, out) == 0, gp.last_error()
        gp.check()
        torch.cuda.synchronize()
        _assert_same(out, ref)


def test_noalloc_rejects_batches_above_its_scratch(P):
    """A batch whose workspace exceeds GPO_NOALLOC_SCRATCH_BYTES is refused before any
    launch (only host-side sizes are read; nothing is dereferenced)."""
    b = W.make_batch(W.CONFIGS["math"].scaled(2))
    gp = P.GraphPO(kappa=b["kappa"], w=b["w"], lambda_eff=b["lambda_eff"])
    db = P.Batch.from_arrays(b, device="cuda")
    out = gp.alloc_outputs(db)
    B = P.binding
    cb = db.c_struct()
    cb.num_states = 1 << 24
    cb.max_states_per_group = 4096
    co = B.COutputs(out["adv"].data_ptr(), None, None, None, None, None, None)
    import torch
    code = P.load().gpo_compute_noalloc(gp._h, ctypes.byref(cb), ctypes.byref(co),
                                        ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert code == 8, code
    assert "built-in scratch" in gp.last_error()
