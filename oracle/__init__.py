"""CPU oracle for GraphPO's advantage construction -- test infrastructure only.

Only the tests, `__graft_entry__.smoke()` and the benchmark's CPU-baseline leg
use this package.  The product path (`paper_2606_18954_gb300`) never imports it.
`build()` compiles `oracle.c` with the host C compiler into `oracle/_build/`.
"""
from __future__ import annotations

import contextlib
import ctypes
import os
import shutil
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")
_lock = threading.Lock()
_lib = None

ERRORS = {0: "ok", 1: "invalid argument", 2: "shape", 3: "bad reward", 4: "non-finite", 5: "no memory"}


class OracleError(RuntimeError):
    def __init__(self, code):
        super().__init__(f"oracle error {code}: {ERRORS.get(code, '?')}")
        self.code = code


class _Batch(ctypes.Structure):
    _fields_ = [
        ("num_groups", ctypes.c_int32), ("num_rollouts", ctypes.c_int32),
        ("num_states", ctypes.c_int32), ("d", ctypes.c_int32),
        ("emb_is_bf16", ctypes.c_int32), ("emb_row_stride", ctypes.c_int64),
        ("total_tokens", ctypes.c_int64),
        ("group_rollout_off", ctypes.c_void_p), ("rollout_step_off", ctypes.c_void_p),
        ("step_len", ctypes.c_void_p), ("rollout_token_off", ctypes.c_void_p),
        ("emb", ctypes.c_void_p), ("reward", ctypes.c_void_p), ("root_emb", ctypes.c_void_p),
        ("parent", ctypes.c_void_p), ("group_state_off", ctypes.c_void_p),
        ("group_token_off", ctypes.c_void_p),
    ]


class _Params(ctypes.Structure):
    _fields_ = [
        ("kappa", ctypes.c_double), ("w", ctypes.c_double), ("lambda_eff", ctypes.c_double),
        ("std_eps", ctypes.c_double), ("std_ddof", ctypes.c_int32), ("merge_rule", ctypes.c_int32),
    ]


_OUT_FIELDS = [
    # name, dtype, per ("T" token | "N" state | "G" group)
    ("adv", np.float64, "T"), ("adv_cor", np.float64, "T"), ("adv_eff", np.float64, "T"),
    ("eff_mask", np.uint8, "T"), ("class_id", np.int32, "N"), ("node_score", np.float64, "N"),
    ("root_score", np.float64, "G"), ("eta", np.float64, "N"), ("step_reward", np.float64, "N"),
    ("a_cor", np.float64, "N"), ("a_eff_node", np.float64, "N"), ("e_eff", np.float64, "N"),
    ("edge_adv", np.float64, "N"), ("edge_eff_mask", np.uint8, "N"),
    ("cor_group_size", np.int32, "N"), ("eff_tree", np.float64, "G"), ("eff_graph", np.float64, "G"),
]


class _Outputs(ctypes.Structure):
    _fields_ = [(name, ctypes.c_void_p) for name, _, _ in _OUT_FIELDS]


def build(force: bool = False) -> str:
    """Compile the oracle with the host C compiler (gcc, -O2, fp64, no fast-math)."""
    src = os.path.join(_HERE, "oracle.c")
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < max(
            os.path.getmtime(src), os.path.getmtime(os.path.join(_HERE, "oracle.h"))):
        tmp = _LIB_PATH + f".{os.getpid()}.tmp"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-pthread",
                               "-ffp-contract=off", src, "-o", tmp, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            lib.oracle_run.argtypes = [ctypes.POINTER(_Batch), ctypes.POINTER(_Params),
                                       ctypes.POINTER(_Outputs), ctypes.c_int]
            lib.oracle_run.restype = ctypes.c_int
            lib.oracle_validate.argtypes = [ctypes.POINTER(_Batch)]
            lib.oracle_validate.restype = ctypes.c_int
            _lib = lib
    return _lib


@contextlib.contextmanager
def library(path: str):
    """Runs the oracle from another build of its C source (for the tests' mutation
    checks, which compile deliberately broken copies) inside the block."""
    global _lib
    _load()
    with _lock:
        saved = _lib
        lib = ctypes.CDLL(path)
        lib.oracle_run.argtypes = saved.oracle_run.argtypes
        lib.oracle_run.restype = ctypes.c_int
        lib.oracle_validate.argtypes = saved.oracle_validate.argtypes
        lib.oracle_validate.restype = ctypes.c_int
        _lib = lib
    try:
        yield
    finally:
        with _lock:
            _lib = saved


def compile_variant(source: str, out_dir: str) -> str:
    """Compiles C source text of the oracle (the header beside it) like build() does."""
    src = os.path.join(out_dir, "oracle.c")
    with open(src, "w") as f:
        f.write(source)
    shutil.copy(os.path.join(_HERE, "oracle.h"), os.path.join(out_dir, "oracle.h"))
    so = os.path.join(out_dir, "liboracle_variant.so")
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-pthread", "-ffp-contract=off", src, "-o", so,
                           "-lm"])
    return so


def default_params(batch: dict, **kw) -> dict:
    p = dict(kappa=float(batch.get("kappa", 0.92)), w=float(batch.get("w", 0.7)),
             lambda_eff=float(batch.get("lambda_eff", 1.0)), std_eps=1e-6, std_ddof=1,
             merge_rule=0)
    p.update(kw)
    return p


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def _ptr(a):
    return a.ctypes.data if a is not None and a.size else None


def _make_batch(batch: dict, with_root: bool = True):
    """The C batch for a dict batch (chain layout, or tree layout when it has
    "parent"), plus the arrays it points into (kept alive by the caller)."""
    go = _c(batch["group_rollout_off"], np.int32)
    sl = _c(batch["step_len"], np.int32)
    rw = _c(batch["reward"], np.uint8)
    is_bf16 = batch["emb_dtype"] == "bf16"
    emb = _c(batch["emb"], np.uint16 if is_bf16 else np.float32)
    root = batch.get("root_emb") if with_root else None
    if root is not None:
        root = _c(root, np.uint16 if is_bf16 else np.float32)
    G, R, N = len(go) - 1, len(rw), int(emb.shape[0])
    if batch.get("parent") is not None:
        par = _c(batch["parent"], np.int32)
        gs = _c(batch["group_state_off"], np.int32)
        gt = _c(batch["group_token_off"], np.int64)
        so = to = None
        T = int(batch.get("total_tokens", gt[-1] if len(gt) else 0))
    else:
        par = gs = gt = None
        so = _c(batch["rollout_step_off"], np.int32)
        to = _c(batch["rollout_token_off"], np.int64)
        R = len(so) - 1
        T = int(batch.get("total_tokens", to[-1] if len(to) else 0))
    keep = [go, so, sl, to, rw, emb, root, par, gs, gt]

    def off(a):  # offset arrays: never empty, passed whenever present
        return a.ctypes.data if a is not None else None

    b = _Batch(G, R, N, int(emb.shape[1]), int(is_bf16), int(emb.shape[1]), T,
               off(go), off(so), _ptr(sl), off(to), _ptr(emb), _ptr(rw), _ptr(root),
               _ptr(par), off(gs), off(gt))
    return b, keep, dict(T=T, N=N, G=G)


def run(batch: dict, params: dict | None = None, threads: int = 1, want=None) -> dict:
    """Run the oracle on a batch (the dict layout of `workloads.make_batch`, or
    the tree layout of `workloads.make_tree_batch`).

    Returns a dict of numpy arrays for every output in `want` (default: all).
    """
    lib = _load()
    p = default_params(batch) if params is None else dict(default_params(batch), **params)
    b, keep, sizes = _make_batch(batch)
    pp = _Params(p["kappa"], p["w"], p["lambda_eff"], p["std_eps"], int(p["std_ddof"]),
                 int(p["merge_rule"]))
    outs = {}
    o = _Outputs()
    for name, dt, per in _OUT_FIELDS:
        if want is None or name in want:
            arr = np.zeros(max(sizes[per], 1), dtype=dt)[: sizes[per]]
            outs[name] = arr
            setattr(o, name, arr.ctypes.data if sizes[per] else None)
    code = lib.oracle_run(ctypes.byref(b), ctypes.byref(pp), ctypes.byref(o), int(threads))
    del keep
    if code != 0:
        raise OracleError(code)
    return outs


def validate(batch: dict) -> int:
    """Return the oracle's validation code (0 = ok) for a batch."""
    lib = _load()
    b, keep, _ = _make_batch(batch, with_root=False)
    code = lib.oracle_validate(ctypes.byref(b))
    del keep
    return code
