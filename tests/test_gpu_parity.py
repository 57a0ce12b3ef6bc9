"""GPU path (through the C ABI) against the CPU oracle, element by element.

Bar: class ids bit-exact; every fp32 output within |gpu - ref| <= 1e-5 |ref| + 1e-6,
ref = the oracle's fp64 value rounded to fp32 (1e-5 relative is the stated
target; the 1e-6 floor covers values that are exactly 0 in exact arithmetic).
The generator keeps every comparable cosine >= 1e-3 away from kappa, so the
threshold decision is unambiguous at both precisions.
"""
import functools

import numpy as np
import pytest

from batches import from_rollouts
from paper_2606_18954_gb300 import workloads as W

pytestmark = pytest.mark.gpu

RTOL, ATOL = 1e-5, 1e-6


@pytest.fixture(scope="module")
def torch_cuda():
    import torch
    if not torch.cuda.is_available():
        pytest.fail("a CUDA device is required for -m gpu tests")
    return torch


@pytest.fixture(scope="module")
def gp_mod(torch_cuda):
    import paper_2606_18954_gb300 as P
    P.build()
    return P


@functools.lru_cache(maxsize=None)
def batch_of(name, groups=None, seed=None):
    spec = W.CONFIGS[name] if groups is None else W.CONFIGS[name].scaled(groups)
    return W.make_batch(spec, seed=seed)


def oracle_params(b, **kw):
    p = dict(kappa=float(b["kappa"]), w=float(b["w"]), lambda_eff=float(b["lambda_eff"]), std_eps=1e-6,
             std_ddof=1, merge_rule=0)
    p.update(kw)
    return p


def run_gpu(P, b, params, flags=0, components=True, nodes=True):
    import torch
    gp = P.GraphPO(kappa=params["kappa"], w=params["w"], lambda_eff=params["lambda_eff"],
                   std_eps=params["std_eps"], std_ddof=params["std_ddof"], merge_rule=params["merge_rule"],
                   flags=flags)
    db = P.Batch.from_arrays(b, device="cuda")
    out = gp(db, components=components, nodes=nodes)
    gp.check()
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in out.items()}


def assert_close(got, ref64, name):
    ref = np.asarray(ref64, np.float64).astype(np.float32).astype(np.float64)
    got = np.asarray(got, np.float64)
    assert got.shape == ref.shape, (name, got.shape, ref.shape)
    err = np.abs(got - ref)
    tol = RTOL * np.abs(ref) + ATOL
    bad = err > tol
    if bad.any():
        i = int(np.argmax(err / tol))
        raise AssertionError(f"{name}: {int(bad.sum())} of {bad.size} outside tolerance; worst at {i}: "
                             f"gpu {got[i]!r} ref {ref64[i]!r} (err/tol {err[i] / tol[i]:.3g})")


def compare(gpu, ref, label=""):
    np.testing.assert_array_equal(gpu["class_id"], ref["class_id"], err_msg=f"{label} class_id")
    assert_close(gpu["node_score"], ref["node_score"], f"{label} node_score")
    assert_close(gpu["edge_adv"], ref["edge_adv"], f"{label} edge_adv")
    assert_close(gpu["adv"], ref["adv"], f"{label} adv")
    if "adv_cor" in gpu:
        assert_close(gpu["adv_cor"], ref["adv_cor"], f"{label} adv_cor")
        assert_close(gpu["adv_eff"], ref["adv_eff"], f"{label} adv_eff")
        np.testing.assert_array_equal(gpu["eff_mask"], ref["eff_mask"], err_msg=f"{label} eff_mask")


def oracle_run(b, params, threads=8):
    import oracle
    return oracle.run(b, params, threads=threads)


# --------------------------------------------------------------------- scaled configs

SCALED = [("tiny", 8), ("math", 4), ("agentic", 24), ("full", 3), ("wide", 1)]


# fused: a group-resident kernel (bf16 groups <= 384 states on the tensor cores, fp32
# chain-layout groups <= 128 states on the CUDA cores); tiled: the multi-kernel path
# (tensor-core similarity for bf16, CUDA-core for fp32); simt: the multi-kernel CUDA-core
# path for bf16 (fp32 embeddings take the CUDA cores on every path)
PATH_FLAGS = {"fused": 0, "tiled": 2, "simt": 1}


@pytest.mark.parametrize("name,groups", SCALED)
@pytest.mark.parametrize("rule", [0, 1])
@pytest.mark.parametrize("path", ["fused", "tiled", "simt"])
def test_parity_scaled(gp_mod, name, groups, rule, path):
    b = batch_of(name, groups)
    if path == "simt" and b["emb_dtype"] != "bf16":
        pytest.skip("fp32 embeddings: the simt flag selects nothing new (same path as fused)")
    params = oracle_params(b, merge_rule=rule)
    ref = oracle_run(b, params)
    gpu = run_gpu(gp_mod, b, params, flags=PATH_FLAGS[path])
    compare(gpu, ref, f"{name}/{rule}/{path}")


@pytest.mark.parametrize("lam", [0.0, 0.5])
@pytest.mark.parametrize("path", ["fused", "tiled"])
def test_parity_lambda(gp_mod, lam, path):
    b = batch_of("math", 3)
    params = oracle_params(b, lambda_eff=lam)
    compare(run_gpu(gp_mod, b, params, flags=PATH_FLAGS[path]), oracle_run(b, params), f"lambda={lam}")


def test_parity_root_embedding(gp_mod):
    b = dict(batch_of("math", 3))
    rng = np.random.default_rng(5)
    G = len(b["group_rollout_off"]) - 1
    # prompt embeddings near the first-step states' centroid direction of each group, so eta > 0
    so, go = b["rollout_step_off"], b["group_rollout_off"]
    first = so[go[:-1]]
    base = W.bf16_bits_to_f32(b["emb"][first]).astype(np.float64)
    root = base + 0.5 * rng.standard_normal(base.shape) / np.sqrt(base.shape[1])
    b["root_emb"] = W.f32_to_bf16_bits(root.astype(np.float32))
    params = oracle_params(b)
    ref = oracle_run(b, params)
    assert np.any(ref["eta"][first] > 0)
    for path in ("fused", "tiled"):
        compare(run_gpu(gp_mod, b, params, flags=PATH_FLAGS[path]), ref, f"root_emb/{path}")


@pytest.mark.parametrize("path", ["fused", "tiled"])
def test_deterministic(gp_mod, path):
    b = batch_of("math", 4)
    params = oracle_params(b)
    a1 = run_gpu(gp_mod, b, params, flags=PATH_FLAGS[path])
    a2 = run_gpu(gp_mod, b, params, flags=PATH_FLAGS[path])
    for k in a1:
        np.testing.assert_array_equal(a1[k], a2[k], err_msg=k)


# --------------------------------------------------------------------- edge cases


def _group(rng, n_roll, steps, d, share=None):
    """One group; `share` maps (rollout, step) -> a shared direction index."""
    dirs = rng.standard_normal((8, d))
    rolls = []
    for r in range(n_roll):
        rows = []
        for h in range(steps if np.isscalar(steps) else steps[r]):
            if share is not None and share(r, h) is not None:
                rows.append(dirs[share(r, h)] + 0.01 * rng.standard_normal(d) / np.sqrt(d))
            else:
                rows.append(rng.standard_normal(d))
        rolls.append((rows, list(rng.integers(1, 40, size=len(rows))), int(rng.integers(0, 2))))
    return rolls


def _margin_ok(b, kappa):
    from batches import emb_f64, states_of
    roll, _, grp = states_of(b)
    Z = emb_f64(b)
    Zn = Z / np.maximum(np.linalg.norm(Z, axis=1), 1e-300)[:, None]
    C = Zn @ Zn.T
    m = (roll[:, None] != roll[None, :]) & (grp[:, None] == grp[None, :])
    return not np.any(np.abs(C[m] - kappa) < 1e-3)


EDGE_CASES = {
    # one group per tile-boundary size (128 rows, 256 columns), plus ragged tails
    "n128": lambda rng: [_group(rng, 8, 16, 128, lambda r, h: h % 3 if h % 2 == 0 else None)],
    "n129": lambda rng: [_group(rng, 3, [43, 43, 43], 128, lambda r, h: 1 if h == 5 else None)],
    "n257": lambda rng: [_group(rng, 5, [51, 52, 51, 51, 52], 64, lambda r, h: h % 4 if h < 8 else None)],
    "n384": lambda rng: [_group(rng, 12, 32, 64, lambda r, h: (h // 4) % 8 if h % 3 == 0 else None)],
    "n700": lambda rng: [_group(rng, 7, 100, 64, lambda r, h: (h // 10) % 8 if h % 2 else None)],
    "mixed": lambda rng: [_group(rng, 2, 3, 64), [], _group(rng, 1, 5, 64),
                          _group(rng, 6, [1, 2, 3, 4, 5, 6], 64, lambda r, h: 0 if h == 0 else None)],
    "one_class": lambda rng: [_group(rng, 10, 6, 64, lambda r, h: 2)],
    "d72": lambda rng: [_group(rng, 5, 7, 72, lambda r, h: h % 2), _group(rng, 4, 9, 72, lambda r, h: 3)],
}


@pytest.mark.parametrize("case", sorted(EDGE_CASES))
@pytest.mark.parametrize("path", ["fused", "tiled", "simt"])
def test_edge_cases(gp_mod, case, path):
    rng = np.random.default_rng(sum(map(ord, case)))
    b = from_rollouts(EDGE_CASES[case](rng), dtype="bf16", kappa=0.9, w=0.7, lambda_eff=1.0)
    assert _margin_ok(b, 0.9)
    params = oracle_params(b)
    compare(run_gpu(gp_mod, b, params, flags=PATH_FLAGS[path]), oracle_run(b, params), case)


def test_zero_rows_and_f32(gp_mod):
    rng = np.random.default_rng(3)
    grp = _group(rng, 4, 5, 32, lambda r, h: 1 if h == 2 else None)
    grp[1][0][3] = np.zeros(32)
    b = from_rollouts([grp, _group(rng, 3, 2, 32)], dtype="f32", kappa=0.9)
    params = oracle_params(b)
    compare(run_gpu(gp_mod, b, params), oracle_run(b, params), "f32 zero rows")


@pytest.mark.parametrize("rollouts,d", [(8, 256), (10, 30), (16, 256), (20, 62)])
def test_parity_f32_instances(gp_mod, rollouts, d):
    """The fp32 group-resident kernel's two instances: groups of at most 64 states (48, 60:
    512 threads, the Gram's k range split between the block's halves, whose partial sums
    are added in a fixed order) and of 65..128 states (96, 120: 256 threads).  d = 30 and 62
    are not multiples of 4: those rows sit in a buffer padded to 32 and 64 columns (a row's
    bytes must be a multiple of 16), and the split range ends ragged."""
    import dataclasses
    import torch
    spec = dataclasses.replace(W.CONFIGS["tiny"], rollouts=rollouts, d=d)
    b = W.make_batch(spec, seed=101 + rollouts + d)
    params = oracle_params(b)
    P = gp_mod
    gp = P.GraphPO(kappa=params["kappa"], w=params["w"], lambda_eff=params["lambda_eff"])
    db = P.Batch.from_arrays(b, device="cuda")
    dp = (d + 3) // 4 * 4
    padded = torch.full((db.emb.shape[0], dp), float("nan"), dtype=torch.float32, device="cuda")
    padded[:, :d] = db.emb
    db.emb = padded[:, :d]  # row stride dp, the padding never read
    assert db.c_struct().emb_row_stride == dp
    out = gp(db, components=True, nodes=True)
    gp.check()
    gpu = {k: v.cpu().numpy() for k, v in out.items()}
    compare(gpu, oracle_run(b, params), f"f32 {rollouts}x6 states, d={d}")


def test_largest_group(gp_mod):
    """One group at the 4096-state limit (16 x 16 tiles of 128 x 256)."""
    rng = np.random.default_rng(11)
    b = from_rollouts([_group(rng, 64, 64, 64, lambda r, h: (h // 8) % 8 if h % 4 == 0 else None)],
                      dtype="bf16", kappa=0.9)
    assert _margin_ok(b, 0.9)
    params = oracle_params(b)
    compare(run_gpu(gp_mod, b, params), oracle_run(b, params), "n4096")


# --------------------------------------------------------------------- errors


def _expect_status(P, b, code, host=False, flags=0):
    import torch
    gp = P.GraphPO(flags=flags)
    db = P.Batch.from_arrays(b, device="cuda")
    if host:
        with pytest.raises(P.GraphPOError) as e:
            gp(db)
        assert e.value.code == code
        return
    gp(db)
    with pytest.raises(P.GraphPOError) as e:
        gp.check()
    assert e.value.code == code, gp.last_error()
    # the context stays usable after a device-side error
    ok = P.Batch.from_arrays(batch_of("tiny", 2), device="cuda")
    gp2 = P.GraphPO(kappa=0.9)
    gp2(ok)
    gp2.check()
    torch.cuda.synchronize()


ERR_PATHS = pytest.mark.parametrize("flags", [0, 2], ids=["fused", "tiled"])


@ERR_PATHS
def test_error_bad_reward(gp_mod, flags):
    b = dict(batch_of("math", 2))
    b["reward"] = b["reward"].copy()
    b["reward"][5] = 2
    _expect_status(gp_mod, b, 3, flags=flags)


@ERR_PATHS
def test_error_bad_step_len(gp_mod, flags):
    b = dict(batch_of("math", 2))
    b["step_len"] = b["step_len"].copy()
    b["step_len"][7] = 0
    _expect_status(gp_mod, b, 2, flags=flags)


@ERR_PATHS
def test_error_token_spans(gp_mod, flags):
    b = dict(batch_of("math", 2))
    b["rollout_token_off"] = b["rollout_token_off"].copy()
    b["rollout_token_off"][3] += 1
    _expect_status(gp_mod, b, 2, flags=flags)


@ERR_PATHS
def test_error_offsets_out_of_range(gp_mod, flags):
    b = dict(batch_of("math", 2))
    b["rollout_step_off"] = b["rollout_step_off"].copy()
    b["rollout_step_off"][4] = 10 ** 6
    _expect_status(gp_mod, b, 2, flags=flags)


@ERR_PATHS
def test_error_nonfinite(gp_mod, flags):
    b = dict(batch_of("math", 2))
    b["emb"] = b["emb"].copy()
    b["emb"][9, 17] = 0x7FC0  # bf16 quiet NaN
    _expect_status(gp_mod, b, 4, flags=flags)


def test_error_group_too_large(gp_mod):
    rng = np.random.default_rng(2)
    b = from_rollouts([_group(rng, 2, 2100, 16)], dtype="bf16")
    _expect_status(gp_mod, b, 5, host=True)


@ERR_PATHS
def test_error_group_above_declared_max(gp_mod, flags):
    """A group larger than the batch's declared max_states_per_group is refused on the device."""
    import dataclasses
    import torch
    P = gp_mod
    db = P.Batch.from_arrays(batch_of("math", 2), device="cuda")
    db = dataclasses.replace(db, max_states_per_group=db.max_states_per_group - 40)
    gp = P.GraphPO(flags=flags)
    gp(db)
    with pytest.raises(P.GraphPOError) as e:
        gp.check()
    assert e.value.code == 5, gp.last_error()
    torch.cuda.synchronize()


def test_error_workspace_too_small(gp_mod):
    import torch
    P = gp_mod
    gp = P.GraphPO()
    db = P.Batch.from_arrays(batch_of("math", 2), device="cuda")
    out = gp.alloc_outputs(db)
    small = torch.empty(1024, dtype=torch.uint8, device="cuda")
    with pytest.raises(P.GraphPOError) as e:
        gp.compute_into(db, out, workspace=small)
    assert e.value.code == 8


# --------------------------------------------------------------------- full-size configs


@pytest.mark.parametrize("name", ["math", "agentic", "full", "wide"])
def test_full_size_whole_batch(gp_mod, name):
    """Whole config on the GPU in the benchmark's launch configuration, every output of
    every group against the oracle (16 host threads; the wide groups' dense fp64
    similarities take the oracle about 3 s per group and thread)."""
    b = batch_of(name)
    params = oracle_params(b)
    compare(run_gpu(gp_mod, b, params), oracle_run(b, params, threads=16), f"{name} whole batch")


@pytest.mark.parametrize("name", ["wide", "full"])
def test_full_size_properties(gp_mod, name):
    """Properties that hold at any size, on the whole config in the benchmark's launch
    configuration."""
    b = batch_of(name)
    params = oracle_params(b)
    gpu = run_gpu(gp_mod, b, params, components=False)
    # properties that hold everywhere: every token of an edge carries the edge's value
    np.testing.assert_array_equal(gpu["adv"], np.repeat(gpu["edge_adv"], b["step_len"]))
    assert np.all(np.isfinite(gpu["adv"]))
    assert np.all((gpu["node_score"] >= 0) & (gpu["node_score"] <= 1))
