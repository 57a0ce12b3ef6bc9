"""Group ranges (gpo_compute_groups) and the pipelined host entry point.

A range call runs the same kernels as a whole-batch call on a subset of the
groups, so the outputs of a set of range calls that covers the batch must equal
the whole-batch outputs bit for bit; the whole-batch outputs themselves are
checked against the oracle in test_gpu_parity.py (and here once more, through
the host entry point, against the oracle).
"""
import numpy as np
import pytest

from paper_2606_18954_gb300 import workloads as W

pytestmark = pytest.mark.gpu

KEYS = ("adv", "adv_cor", "adv_eff", "eff_mask", "class_id", "node_score", "edge_adv", "edge_cor", "edge_eff",
        "edge_eff_mask", "group_eff", "group_eff_graph")


@pytest.fixture(scope="module")
def P():
    import torch
    if not torch.cuda.is_available():
        pytest.fail("a CUDA device is required for -m gpu tests")
    import paper_2606_18954_gb300 as P
    P.build()
    return P


def _batch(name, groups):
    return W.make_batch(W.CONFIGS[name].scaled(groups))


def _gp(P, b, flags=0):
    return P.GraphPO(kappa=b["kappa"], w=b["w"], lambda_eff=b["lambda_eff"], flags=flags)


@pytest.mark.parametrize("name", ["math", "tiny"])  # bf16 and fp32 group-resident paths
@pytest.mark.parametrize("cuts", [(0, 3, 5, 8), (0, 1, 8), (0, 8)], ids=["3-2-3", "1-7", "whole"])
def test_ranges_cover_batch(P, cuts, name):
    import torch
    b = _batch(name, 8)
    gp = _gp(P, b)
    db = P.Batch.from_arrays(b, device="cuda")
    ref = gp(db, components=True, nodes=True, edges=True, efficiency=True)
    gp.check()
    out = gp.alloc_outputs(db, components=True, nodes=True, edges=True, efficiency=True)
    for v in out.values():
        v.fill_(-7)  # every element must be overwritten
    ws = gp.workspace(db)
    stream = torch.cuda.current_stream()
    gp.compute_groups(db, out, 0, 0, True, ws, stream)
    for a, c in zip(cuts[:-1], cuts[1:]):
        gp.compute_groups(db, out, a, c - a, False, ws, stream)
    gp.check()
    for k in KEYS:
        assert torch.equal(out[k], ref[k]), k


def test_ranges_on_parallel_streams(P):
    import torch
    b = _batch("agentic", 24)
    gp = _gp(P, b)
    db = P.Batch.from_arrays(b, device="cuda")
    ref = gp(db)
    gp.check()
    out = gp.alloc_outputs(db)
    out["adv"].fill_(-7)
    ws = gp.workspace(db)
    main = torch.cuda.current_stream()
    gp.compute_groups(db, out, 0, 0, True, ws, main)
    ev = torch.cuda.Event()
    ev.record(main)
    streams = [torch.cuda.Stream() for _ in range(3)]
    for i, s in enumerate(streams):
        s.wait_event(ev)
        gp.compute_groups(db, out, 8 * i, 8, False, ws, s)
        main.wait_stream(s)
    gp.check(main)
    assert torch.equal(out["adv"], ref["adv"])


def test_range_error_reported_after_last_range(P):
    import torch
    b = dict(_batch("math", 4))
    b["reward"] = b["reward"].copy()
    b["reward"][-1] = 2  # a rollout of the last group
    gp = _gp(P, b)
    db = P.Batch.from_arrays(b, device="cuda")
    out = gp.alloc_outputs(db)
    ws = gp.workspace(db)
    s = torch.cuda.current_stream()
    gp.compute_groups(db, out, 0, 0, True, ws, s)
    gp.compute_groups(db, out, 0, 2, False, ws, s)
    gp.compute_groups(db, out, 2, 2, False, ws, s)
    with pytest.raises(P.GraphPOError) as e:
        gp.check()
    assert e.value.code == 3


def test_range_argument_checks(P):
    import torch
    b = _batch("math", 4)
    db = P.Batch.from_arrays(b, device="cuda")
    gp = _gp(P, b)
    out = gp.alloc_outputs(db)
    ws = gp.workspace(db)
    s = torch.cuda.current_stream()
    for a, n in [(-1, 1), (3, 2), (5, 0), (0, -1)]:
        with pytest.raises(P.GraphPOError) as e:
            gp.compute_groups(db, out, a, n, False, ws, s)
        assert e.value.code == 1
    tiled = _gp(P, b, flags=P.FLAG_TILED)
    with pytest.raises(P.GraphPOError) as e:  # a partial range needs the group-resident path
        tiled.compute_groups(db, out, 1, 2, True, ws, s)
    assert e.value.code == 5
    tiled.compute_groups(db, out, 0, 4, True, ws, s)  # the whole batch is fine on any path
    tiled.check()
    torch.cuda.synchronize()


@pytest.mark.parametrize("chunk_bytes", [1 << 20, 1 << 40], ids=["pipelined", "single"])
def test_compute_host_matches_oracle(P, chunk_bytes):
    import torch
    import oracle
    b = _batch("math", 12)
    gp = _gp(P, b)
    hb = P.Batch.from_arrays(b, device="cpu", pin=True)
    out = gp.compute_host(hb, chunk_bytes=chunk_bytes)
    db = P.Batch.from_arrays(b, device="cuda")
    ref = gp(db)
    gp.check()
    assert torch.equal(out, ref["adv"].cpu())
    o = oracle.run(b, dict(kappa=b["kappa"], w=b["w"], lambda_eff=b["lambda_eff"]), threads=8, want={"adv"})
    want = o["adv"].astype(np.float32)
    got = out.numpy()
    assert np.all(np.abs(got - want) <= 1e-5 * np.abs(want) + 1e-6)


def test_compute_host_tree_layout_pipelined(P):
    """compute_host over chunks of a tree-layout batch (token spans per group) against the
    device-resident call."""
    import torch
    b = W.make_tree_batch(W.TREE_CONFIGS["tree"].scaled(groups=8))
    gp = _gp(P, b)
    hb = P.Batch.from_arrays(b, device="cpu", pin=True)
    out = gp.compute_host(hb, chunk_bytes=1 << 19)  # 3.4 MB of embeddings: six chunks
    again = gp.compute_host(hb, chunk_bytes=1 << 19)  # staging buffers reused
    ref = gp(P.Batch.from_arrays(b, device="cuda"))
    gp.check()
    assert torch.equal(out, ref["adv"].cpu()) and torch.equal(again, out)


@pytest.mark.gpu
def test_compute_host_argument_checks(P):
    """gpo_compute_host refuses host and device batches of different sizes, and a NULL host array."""
    import ctypes
    import torch
    b = W.make_batch(W.CONFIGS["math"].scaled(2))
    gp = P.GraphPO(kappa=b["kappa"], w=b["w"], lambda_eff=b["lambda_eff"])
    hb = P.Batch.from_arrays(b, device="cpu", pin=True)
    db = P.Batch.from_arrays(b, device="cuda")
    out = gp.alloc_outputs(db)
    ws = gp.workspace(db)
    host_adv = torch.empty(hb.total_tokens, dtype=torch.float32, pin_memory=True)
    L = P.binding.load()
    co = P.binding._c_outputs(out)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)

    def call(h, d, adv_ptr):
        return L.gpo_compute_host(gp._h, ctypes.byref(h), ctypes.byref(d), ctypes.byref(co), adv_ptr, 0,
                                  ws.data_ptr(), ws.numel(), stream)

    h, d = hb.c_struct(), db.c_struct()
    h.total_tokens += 1
    assert call(h, d, host_adv.data_ptr()) == 1
    h = hb.c_struct()
    h.emb_row_stride += 8
    assert call(h, d, host_adv.data_ptr()) == 1
    assert call(hb.c_struct(), d, None) == 1  # no host output
    h = hb.c_struct()
    h.step_len = None
    assert call(h, d, host_adv.data_ptr()) == 1
    # a correct call on the same context afterwards
    assert call(hb.c_struct(), d, host_adv.data_ptr()) == 0
    gp.check()
    ref = gp(db)["adv"].cpu()
    torch.cuda.synchronize()
    assert torch.equal(host_adv, ref)


@pytest.mark.gpu
def test_compute_host_pageable_memory(P):
    """Host arrays in pageable memory (no pinning): same advantages, one upload at a time."""
    b = W.make_batch(W.CONFIGS["math"].scaled(4))
    gp = P.GraphPO(kappa=b["kappa"], w=b["w"], lambda_eff=b["lambda_eff"])
    hb = P.Batch.from_arrays(b, device="cpu", pin=False)
    out = gp.compute_host(hb, chunk_bytes=1 << 20)
    ref = gp(P.Batch.from_arrays(b, device="cuda"))["adv"].cpu()
    assert (out == ref).all()
