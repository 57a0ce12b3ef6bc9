"""The small parity cases under the debug build of libgraphpo.

`compute-sanitizer` is not available here, so the library has a debug build of its own
(GPO_DEBUG, buildlib.build(debug=True)): every kernel checks the indices of its global
output writes, of the compensated statistics' rows, of the similarity stage's norms and
spanning-forest edges and of the fp32 kernel's shared-memory rows before it uses them, and
reports GPO_ERR_BOUNDS (skipping the access) instead of touching memory outside an array.
This test builds that library and runs, in a child process that loads it (GRAPHPO_LIB),
scaled batches of every shape through every path against the oracle, plus a policy-loss
call: each must finish with no error status and within the parity bar.
"""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r'''
import sys
import numpy as np
import torch
sys.path.insert(0, ROOT)
import oracle
import paper_2606_18954_gb300 as P
from paper_2606_18954_gb300 import binding, buildlib, workloads as W
assert binding.lib_path() == buildlib.DEBUG_LIB, binding.lib_path()
assert b"GPO_DEBUG" in binding.load().gpo_version(), binding.load().gpo_version()

def check(b, flags, what):
    params = dict(kappa=float(b["kappa"]), w=float(b["w"]), lambda_eff=float(b["lambda_eff"]))
    gp = P.GraphPO(flags=flags, **params)
    out = gp(P.Batch.from_arrays(b, device="cuda"), nodes=True)
    gp.check()  # raises on any device status, GPO_ERR_BOUNDS included
    ref = oracle.run(b, params, threads=8)
    assert np.array_equal(out["class_id"].cpu().numpy(), ref["class_id"]), what
    r = ref["adv"].astype(np.float32).astype(np.float64)
    err = np.abs(out["adv"].cpu().numpy().astype(np.float64) - r)
    assert np.all(err <= 1e-5 * np.abs(r) + 1e-6), (what, float(err.max()))
    print("ok", what, flush=True)

cases = [("tiny", 4, (0, 2)), ("math", 2, (0, 2, 1)), ("agentic", 8, (0, 2)), ("full", 2, (0, 2)),
         ("wide", 1, (2,))]
for name, groups, paths in cases:
    b = W.make_batch(W.CONFIGS[name].scaled(groups))
    for flags in paths:
        check(b, flags, f"{name} flags={flags}")
tb = W.make_tree_batch(W.TREE_CONFIGS["tree"].scaled(3))
for flags in (0, 2):
    check(tb, flags, f"tree flags={flags}")
# the policy loss on the device advantages of the last chain batch
b = W.make_batch(W.CONFIGS["math"].scaled(2))
gp = P.GraphPO(kappa=float(b["kappa"]), w=float(b["w"]), lambda_eff=float(b["lambda_eff"]))
db = P.Batch.from_arrays(b, device="cuda")
out = gp(db, nodes=True)
lp = W.make_logprobs(db.total_tokens, 5)
t = lambda x: torch.from_numpy(np.ascontiguousarray(x)).cuda()
res = gp.token_loss(db, gp.loss_plan(db), t(lp["logp"]), t(lp["old_logp"]), edge_adv=out["edge_adv"])
gp.check()
assert np.isfinite(float(res["loss"].cpu()[0]))
print("ok loss", flush=True)
'''


def test_parity_under_debug_build():
    import torch
    if not torch.cuda.is_available():
        pytest.fail("a CUDA device is required for -m gpu tests")
    from paper_2606_18954_gb300 import buildlib
    lib = buildlib.build(debug=True)
    env = dict(os.environ, GRAPHPO_LIB=lib)
    r = subprocess.run([sys.executable, "-c", f"ROOT = {ROOT!r}\n" + CHILD], env=env, capture_output=True, text=True,
                       timeout=900)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-3000:]
    assert r.stdout.count("ok ") == 13, r.stdout
