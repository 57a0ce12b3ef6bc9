"""ctypes binding of libgraphpo (include/graphpo.h).

Argument marshalling only: every step of the path runs in the library's CUDA
kernels.  PyTorch supplies device memory (inputs, outputs, workspace) and the
current CUDA stream.  There is no CPU fallback: if the library is not built or
no sm_103 GPU is present the calls raise.
"""
from __future__ import annotations

import ctypes
import dataclasses
import os
import threading
from typing import Optional

import numpy as np

from . import buildlib as _build

GPO_OK = 0
STATUS_NAMES = {0: "ok", 1: "invalid argument", 2: "shape", 3: "bad reward", 4: "non-finite",
                5: "unsupported", 6: "cuda", 7: "timeout", 8: "workspace"}
MERGE_RULES = {"noncausal": 0, "same_depth": 1}
FLAG_SIMT_SIMILARITY = 1
FLAG_TILED = 2
FLAG_DEBUG_TIMEOUT = 4  # tests of the failure path: the tensor-core kernels' first wait runs out
EMB_BF16, EMB_F32 = 0, 1


class GraphPOError(RuntimeError):
    def __init__(self, code: int, msg: str = ""):
        super().__init__(f"graphpo status {code} ({STATUS_NAMES.get(code, '?')}): {msg}")
        self.code = code


class Params(ctypes.Structure):
    _fields_ = [("kappa", ctypes.c_double), ("w", ctypes.c_double), ("lambda_eff", ctypes.c_double),
                ("std_eps", ctypes.c_double), ("std_ddof", ctypes.c_int32), ("merge_rule", ctypes.c_int32),
                ("flags", ctypes.c_int32)]


class CBatch(ctypes.Structure):
    _fields_ = [("num_groups", ctypes.c_int32), ("num_rollouts", ctypes.c_int32),
                ("num_states", ctypes.c_int32), ("d", ctypes.c_int32), ("emb_dtype", ctypes.c_int32),
                ("max_states_per_group", ctypes.c_int32), ("emb_row_stride", ctypes.c_int64),
                ("total_tokens", ctypes.c_int64),
                ("group_rollout_off", ctypes.c_void_p), ("rollout_step_off", ctypes.c_void_p),
                ("step_len", ctypes.c_void_p), ("rollout_token_off", ctypes.c_void_p),
                ("emb", ctypes.c_void_p), ("reward", ctypes.c_void_p), ("root_emb", ctypes.c_void_p),
                ("parent", ctypes.c_void_p), ("group_state_off", ctypes.c_void_p),
                ("group_token_off", ctypes.c_void_p)]


class COutputs(ctypes.Structure):
    _fields_ = [("adv", ctypes.c_void_p), ("adv_cor", ctypes.c_void_p), ("adv_eff", ctypes.c_void_p),
                ("eff_mask", ctypes.c_void_p), ("class_id", ctypes.c_void_p),
                ("node_score", ctypes.c_void_p), ("edge_adv", ctypes.c_void_p), ("edge_cor", ctypes.c_void_p),
                ("edge_eff", ctypes.c_void_p), ("edge_eff_mask", ctypes.c_void_p), ("group_eff", ctypes.c_void_p),
                ("group_eff_graph", ctypes.c_void_p)]

OUTPUT_NAMES = ("adv", "adv_cor", "adv_eff", "eff_mask", "class_id", "node_score", "edge_adv", "edge_cor", "edge_eff",
                "edge_eff_mask", "group_eff", "group_eff_graph")


class LossParams(ctypes.Structure):
    _fields_ = [("clip_low", ctypes.c_double), ("clip_high", ctypes.c_double), ("beta_kl", ctypes.c_double),
                ("lambda_eff", ctypes.c_double), ("form", ctypes.c_int32), ("norm", ctypes.c_int32)]


class LossInputs(ctypes.Structure):
    _fields_ = [(k, ctypes.c_void_p) for k in ("logp", "old_logp", "ref_logp", "edge_adv", "edge_cor", "edge_eff",
                                                "edge_eff_mask")]


class LossOutputs(ctypes.Structure):
    _fields_ = [("loss", ctypes.c_void_p), ("grad_logp", ctypes.c_void_p), ("stats", ctypes.c_void_p)]


LOSS_FORMS = {"dual": 0, "split": 1}
LOSS_NORMS = {"edge": 0, "token": 1}
LOSS_NSTATS = 4

EXPORTS = ["gpo_create", "gpo_workspace_size", "gpo_compute", "gpo_sync_status", "gpo_status_string",
           "gpo_last_error", "gpo_version", "gpo_destroy", "gpo_enable_timing", "gpo_stage_times", "gpo_compute_noalloc",
           "gpo_compute_groups", "gpo_compute_host", "gpo_loss_plan_size", "gpo_loss_plan", "gpo_token_loss",
           "gpo_layer_budget"]

FUSED_MAX_STATES = 384  # largest group the group-resident path (and gpo_compute_groups) serves

_lib = None
_lock = threading.Lock()


def lib_path() -> str:
    """The library this process loads: GRAPHPO_LIB if set (e.g. the debug build,
    buildlib.DEBUG_LIB), else the in-tree release build."""
    return os.environ.get("GRAPHPO_LIB") or _build.LIB


def load(build_if_missing: bool = False):
    """Load libgraphpo.so (optionally building it first)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = lib_path()
        if not os.path.exists(path):
            if not build_if_missing:
                raise RuntimeError(f"{path} is missing: build it with paper_2606_18954_gb300.build()")
            _build.build()
        L = ctypes.CDLL(path)
        L.gpo_create.argtypes = [ctypes.POINTER(ctypes.c_void_p), ctypes.POINTER(Params)]
        L.gpo_create.restype = ctypes.c_int
        L.gpo_workspace_size.argtypes = [ctypes.c_void_p, ctypes.POINTER(CBatch), ctypes.POINTER(ctypes.c_size_t)]
        L.gpo_workspace_size.restype = ctypes.c_int
        L.gpo_compute.argtypes = [ctypes.c_void_p, ctypes.POINTER(CBatch), ctypes.POINTER(COutputs),
                                  ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p]
        L.gpo_compute.restype = ctypes.c_int
        L.gpo_compute_groups.argtypes = [ctypes.c_void_p, ctypes.POINTER(CBatch), ctypes.POINTER(COutputs),
                                         ctypes.c_int64, ctypes.c_int64, ctypes.c_int, ctypes.c_void_p,
                                         ctypes.c_size_t, ctypes.c_void_p]
        L.gpo_compute_groups.restype = ctypes.c_int
        L.gpo_compute_host.argtypes = [ctypes.c_void_p, ctypes.POINTER(CBatch), ctypes.POINTER(CBatch),
                                       ctypes.POINTER(COutputs), ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p,
                                       ctypes.c_size_t, ctypes.c_void_p]
        L.gpo_compute_host.restype = ctypes.c_int
        L.gpo_sync_status.argtypes = [ctypes.c_void_p, ctypes.c_void_p]
        L.gpo_sync_status.restype = ctypes.c_int
        L.gpo_status_string.argtypes = [ctypes.c_int]
        L.gpo_status_string.restype = ctypes.c_char_p
        L.gpo_last_error.argtypes = [ctypes.c_void_p]
        L.gpo_last_error.restype = ctypes.c_char_p
        L.gpo_version.argtypes = []
        L.gpo_version.restype = ctypes.c_char_p
        L.gpo_destroy.argtypes = [ctypes.c_void_p]
        L.gpo_destroy.restype = None
        L.gpo_compute_noalloc.argtypes = [ctypes.c_void_p, ctypes.POINTER(CBatch), ctypes.POINTER(COutputs),
                                          ctypes.c_void_p]
        L.gpo_compute_noalloc.restype = ctypes.c_int
        L.gpo_enable_timing.argtypes = [ctypes.c_void_p, ctypes.c_int]
        L.gpo_enable_timing.restype = ctypes.c_int
        L.gpo_stage_times.argtypes = [ctypes.c_void_p, ctypes.POINTER(ctypes.c_float),
                                      ctypes.POINTER(ctypes.c_char_p), ctypes.c_int, ctypes.POINTER(ctypes.c_int)]
        L.gpo_stage_times.restype = ctypes.c_int
        L.gpo_layer_budget.argtypes = [ctypes.c_void_p, ctypes.POINTER(CBatch), ctypes.c_int32, ctypes.c_int32,
                                       ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                       ctypes.c_size_t, ctypes.c_void_p]
        L.gpo_layer_budget.restype = ctypes.c_int
        L.gpo_loss_plan_size.argtypes = [ctypes.POINTER(CBatch), ctypes.POINTER(ctypes.c_size_t)]
        L.gpo_loss_plan_size.restype = ctypes.c_int
        L.gpo_loss_plan.argtypes = [ctypes.c_void_p, ctypes.POINTER(CBatch), ctypes.c_void_p, ctypes.c_size_t,
                                    ctypes.c_void_p]
        L.gpo_loss_plan.restype = ctypes.c_int
        L.gpo_token_loss.argtypes = [ctypes.c_void_p, ctypes.POINTER(CBatch), ctypes.c_void_p,
                                     ctypes.POINTER(LossParams), ctypes.POINTER(LossInputs),
                                     ctypes.POINTER(LossOutputs), ctypes.c_void_p]
        L.gpo_token_loss.restype = ctypes.c_int
        _lib = L
        return L


def workspace_size(batch, ctx=None) -> int:
    """Device workspace bytes of gpo_compute for this batch (a `Batch`, or a `CBatch`).
    Reads only the batch's host-side sizes, pointer nullness and alignment: no device
    is needed without a context."""
    L = load()
    cb = batch if isinstance(batch, CBatch) else batch.c_struct()
    n = ctypes.c_size_t()
    code = L.gpo_workspace_size(ctx, ctypes.byref(cb), ctypes.byref(n))
    if code != GPO_OK:
        raise GraphPOError(code, L.gpo_last_error(ctx).decode() if ctx else "gpo_workspace_size")
    return n.value


def loss_plan_size(batch) -> int:
    """Device bytes of the token-loss plan for this batch (no device needed)."""
    L = load()
    cb = batch if isinstance(batch, CBatch) else batch.c_struct()
    n = ctypes.c_size_t()
    code = L.gpo_loss_plan_size(ctypes.byref(cb), ctypes.byref(n))
    if code != GPO_OK:
        raise GraphPOError(code, "gpo_loss_plan_size")
    return n.value


def _ptr(t) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _c_outputs(out: dict) -> COutputs:
    return COutputs(*[_ptr(out.get(k)) if out.get(k) is not None and out[k].numel() else None
                      for k in OUTPUT_NAMES])


@dataclasses.dataclass
class Batch:
    """Device tensors of one batch (see include/graphpo.h).  Chain layout: every rollout a
    path from the prompt root (rollout_step_off, rollout_token_off).  Tree layout
    (`parent` given): states in depth-first pre-order per group, parent = group-local
    index of p(v) or -1, leaves = rollouts (group_state_off, group_token_off); the
    chain-only offsets are then None."""
    group_rollout_off: "torch.Tensor"   # int32 [G+1]
    rollout_step_off: "Optional[torch.Tensor]"   # int32 [R+1] (chain layout)
    step_len: "torch.Tensor"            # int32 [N]
    rollout_token_off: "Optional[torch.Tensor]"  # int64 [R+1] (chain layout)
    emb: "torch.Tensor"                 # bf16 or fp32 [N, d], unit stride in d
    reward: "torch.Tensor"              # uint8 [R]
    total_tokens: int
    max_states_per_group: int
    root_emb: "Optional[torch.Tensor]" = None
    parent: "Optional[torch.Tensor]" = None           # int32 [N] (tree layout)
    group_state_off: "Optional[torch.Tensor]" = None  # int32 [G+1] (tree layout)
    group_token_off: "Optional[torch.Tensor]" = None  # int64 [G+1] (tree layout)

    @property
    def is_tree(self):
        return self.parent is not None

    @property
    def num_groups(self):
        return self.group_rollout_off.numel() - 1

    @property
    def num_rollouts(self):
        return self.reward.numel() if self.is_tree else self.rollout_step_off.numel() - 1

    @property
    def num_states(self):
        return self.emb.shape[0]

    def c_struct(self) -> CBatch:
        import torch
        e = self.emb
        assert e.dim() == 2 and (e.numel() == 0 or e.stride(1) == 1), "embeddings must be [N, d] with unit inner stride"
        dt = EMB_BF16 if e.dtype == torch.bfloat16 else EMB_F32
        if e.dtype not in (torch.bfloat16, torch.float32):
            raise TypeError("embeddings must be bfloat16 or float32")
        return CBatch(self.num_groups, self.num_rollouts, e.shape[0], e.shape[1], dt,
                      int(self.max_states_per_group), e.stride(0) if e.shape[0] > 1 else e.shape[1],
                      int(self.total_tokens),
                      _ptr(self.group_rollout_off), _ptr(self.rollout_step_off),
                      _ptr(self.step_len) if self.step_len.numel() else None, _ptr(self.rollout_token_off),
                      _ptr(e) if e.numel() else None, _ptr(self.reward) if self.reward.numel() else None,
                      _ptr(self.root_emb),
                      _ptr(self.parent) if self.parent is not None and self.parent.numel() else None,
                      _ptr(self.group_state_off), _ptr(self.group_token_off))

    @staticmethod
    def from_arrays(arrs: dict, device="cuda", pin: bool = False) -> "Batch":
        """From the numpy dict layout of `workloads.make_batch` or `workloads.make_tree_batch`
        (copied to `device`)."""
        import torch

        def t(a, dt):
            x = torch.from_numpy(np.ascontiguousarray(a).astype(dt, copy=False))
            if pin and device == "cpu":
                x = x.pin_memory()
            return x.to(device) if device != "cpu" else x

        if arrs["emb_dtype"] == "bf16":
            emb = t(np.asarray(arrs["emb"], np.uint16).view(np.int16), np.int16).view(torch.bfloat16)
            root = arrs.get("root_emb")
            root = t(np.asarray(root, np.uint16).view(np.int16), np.int16).view(torch.bfloat16) if root is not None else None
        else:
            emb = t(arrs["emb"], np.float32)
            root = arrs.get("root_emb")
            root = t(root, np.float32) if root is not None else None
        go = np.asarray(arrs["group_rollout_off"])
        if arrs.get("parent") is not None:
            gso = np.asarray(arrs["group_state_off"])
            gto = np.asarray(arrs["group_token_off"])
            ng = np.diff(gso)
            return Batch(t(go, np.int32), None, t(arrs["step_len"], np.int32), None, emb,
                         t(arrs["reward"], np.uint8), int(gto[-1]) if len(gto) else 0,
                         int(ng.max()) if len(ng) else 0, root, parent=t(arrs["parent"], np.int32),
                         group_state_off=t(gso, np.int32), group_token_off=t(gto, np.int64))
        so = np.asarray(arrs["rollout_step_off"])
        ng = so[go[1:]] - so[go[:-1]] if len(go) > 1 else np.zeros(0)
        return Batch(t(go, np.int32), t(so, np.int32), t(arrs["step_len"], np.int32),
                     t(arrs["rollout_token_off"], np.int64), emb, t(arrs["reward"], np.uint8),
                     int(arrs["rollout_token_off"][-1]) if len(arrs["rollout_token_off"]) else 0,
                     int(ng.max()) if len(ng) else 0, root)

    def to(self, device, non_blocking=False) -> "Batch":
        f = lambda x: None if x is None else x.to(device, non_blocking=non_blocking)
        return Batch(f(self.group_rollout_off), f(self.rollout_step_off), f(self.step_len),
                     f(self.rollout_token_off), f(self.emb), f(self.reward), self.total_tokens,
                     self.max_states_per_group, f(self.root_emb), f(self.parent), f(self.group_state_off),
                     f(self.group_token_off))


class GraphPO:
    """One context of the advantage path on the current CUDA device.

    gp = GraphPO(kappa=0.92, w=0.7, lambda_eff=1.0)
    out = gp(batch)            # dict of device tensors; enqueued on the current stream
    gp.check()                 # waits and raises GraphPOError on a device-side error
    """

    def __init__(self, kappa=0.92, w=0.7, lambda_eff=1.0, std_eps=1e-6, std_ddof=1,
                 merge_rule="noncausal", flags=0):
        self._lib = load()
        self.params = Params(float(kappa), float(w), float(lambda_eff), float(std_eps), int(std_ddof),
                             MERGE_RULES[merge_rule] if isinstance(merge_rule, str) else int(merge_rule),
                             int(flags))
        h = ctypes.c_void_p()
        code = self._lib.gpo_create(ctypes.byref(h), ctypes.byref(self.params))
        if code != GPO_OK:
            raise GraphPOError(code, "gpo_create")
        self._h = h
        self._ws = None

    def close(self):
        if getattr(self, "_h", None) and self._h.value:
            self._lib.gpo_destroy(self._h)
            self._h = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def last_error(self) -> str:
        return self._lib.gpo_last_error(self._h).decode()

    def workspace_size(self, batch: Batch) -> int:
        return workspace_size(batch, self._h)

    def workspace(self, batch: Batch):
        import torch
        need = self.workspace_size(batch)
        if self._ws is None or self._ws.numel() < need or self._ws.device != batch.emb.device:
            self._ws = torch.empty(max(need, 256), dtype=torch.uint8, device=batch.emb.device)
        return self._ws

    def alloc_outputs(self, batch: Batch, components=False, nodes=False, edges=False, efficiency=False) -> dict:
        """Output tensors: per-token A_dual always; `components` adds per-token A_cor, A_eff and
        m_eff; `nodes` class ids, S(v) and per-edge A_dual; `edges` per-edge A_cor, A_eff and
        m_eff (the split loss form's inputs); `efficiency` Eff per group in both readings."""
        import torch
        dev = batch.emb.device
        T, N, G = batch.total_tokens, batch.num_states, batch.num_groups
        out = {"adv": torch.empty(max(T, 1), dtype=torch.float32, device=dev)[:T]}
        if components:
            out["adv_cor"] = torch.empty(max(T, 1), dtype=torch.float32, device=dev)[:T]
            out["adv_eff"] = torch.empty(max(T, 1), dtype=torch.float32, device=dev)[:T]
            out["eff_mask"] = torch.empty(max(T, 4), dtype=torch.uint8, device=dev)[:T]
        if nodes:
            out["class_id"] = torch.empty(max(N, 1), dtype=torch.int32, device=dev)[:N]
            out["node_score"] = torch.empty(max(N, 1), dtype=torch.float32, device=dev)[:N]
            out["edge_adv"] = torch.empty(max(N, 1), dtype=torch.float32, device=dev)[:N]
        if edges:
            out["edge_cor"] = torch.empty(max(N, 1), dtype=torch.float32, device=dev)[:N]
            out["edge_eff"] = torch.empty(max(N, 1), dtype=torch.float32, device=dev)[:N]
            out["edge_eff_mask"] = torch.empty(max(N, 1), dtype=torch.uint8, device=dev)[:N]
        if efficiency:
            out["group_eff"] = torch.empty(max(G, 1), dtype=torch.float32, device=dev)[:G]
            out["group_eff_graph"] = torch.empty(max(G, 1), dtype=torch.float32, device=dev)[:G]
        return out

    def compute_into(self, batch: Batch, out: dict, workspace=None, stream=None) -> None:
        import torch
        ws = self.workspace(batch) if workspace is None else workspace
        if stream is None:
            stream = torch.cuda.current_stream(batch.emb.device)
        co = _c_outputs(out)
        cb = batch.c_struct()
        code = self._lib.gpo_compute(self._h, ctypes.byref(cb), ctypes.byref(co), ws.data_ptr(), ws.numel(),
                                     ctypes.c_void_p(stream.cuda_stream))
        if code != GPO_OK:
            raise GraphPOError(code, self.last_error())

    def compute_groups(self, batch: Batch, out: dict, first_group: int, num_groups: int, clear_status: bool,
                       workspace, stream) -> None:
        """gpo_compute_groups: the path for groups [first_group, first_group + num_groups) of the
        whole `batch` into the whole `out` (see include/graphpo.h)."""
        self._groups_raw(batch.c_struct(), _c_outputs(out), first_group, num_groups, clear_status, workspace, stream)

    def _groups_raw(self, cb, co, first_group, num_groups, clear_status, workspace, stream) -> None:
        code = self._lib.gpo_compute_groups(self._h, ctypes.byref(cb), ctypes.byref(co), int(first_group),
                                            int(num_groups), int(bool(clear_status)), workspace.data_ptr(),
                                            workspace.numel(), ctypes.c_void_p(stream.cuda_stream))
        if code != GPO_OK:
            raise GraphPOError(code, self.last_error())

    def __call__(self, batch: Batch, components=False, nodes=False, edges=False, efficiency=False,
                 stream=None) -> dict:
        out = self.alloc_outputs(batch, components, nodes, edges, efficiency)
        self.compute_into(batch, out, stream=stream)
        return out

    # ---- per-layer graph construction (gpo_layer_budget)

    def layer_budget(self, batch: Batch, layer: int, b_next: int, active=None, classes: bool = False,
                     out=None, workspace=None, stream=None) -> dict:
        """Next-layer budgets (int32 [N]) and optionally the class ids after layer `layer` of a
        tree-layout batch holding the states sampled so far; enqueued on the current stream."""
        import torch
        dev = batch.emb.device
        if stream is None:
            stream = torch.cuda.current_stream(dev)
        N = batch.num_states
        if out is None:
            out = {"budget": torch.empty(max(N, 1), dtype=torch.int32, device=dev)[:N]}
            if classes:
                out["class_id"] = torch.empty(max(N, 1), dtype=torch.int32, device=dev)[:N]
        ws = self.workspace(batch) if workspace is None else workspace
        cb = batch.c_struct()
        ptr = lambda t: None if t is None or t.numel() == 0 else t.data_ptr()
        code = self._lib.gpo_layer_budget(self._h, ctypes.byref(cb), int(layer), int(b_next), ptr(active),
                                          ptr(out["budget"]), ptr(out.get("class_id")), ws.data_ptr(), ws.numel(),
                                          ctypes.c_void_p(stream.cuda_stream))
        if code != GPO_OK:
            raise GraphPOError(code, self.last_error())
        return out

    # ---- policy loss (gpo_loss_plan / gpo_token_loss)

    def loss_plan(self, batch: Batch, plan=None, stream=None):
        """Builds (into `plan`, a uint8 device tensor, allocated if None) the loss plan of the
        batch's structure and returns it; enqueued on the current stream."""
        import torch
        if stream is None:
            stream = torch.cuda.current_stream(batch.step_len.device)
        cb = batch.c_struct()
        need = loss_plan_size(cb)
        if plan is None or plan.numel() < need:
            plan = torch.empty(max(need, 256), dtype=torch.uint8, device=batch.step_len.device)
        code = self._lib.gpo_loss_plan(self._h, ctypes.byref(cb), plan.data_ptr(), plan.numel(),
                                       ctypes.c_void_p(stream.cuda_stream))
        if code != GPO_OK:
            raise GraphPOError(code, self.last_error())
        return plan

    def token_loss(self, batch: Batch, plan, logp, old_logp, ref_logp=None, edge_adv=None, edge_cor=None,
                   edge_eff=None, edge_eff_mask=None, clip_low=0.2, clip_high=0.2, beta_kl=0.0, lambda_eff=1.0,
                   form="dual", norm="edge", grad=True, stats=True, out=None, stream=None) -> dict:
        """gpo_token_loss: returns {"loss": [1] float32, "grad_logp": [T] float32 (if grad),
        "stats": [4] float64 (if stats)} as device tensors (or fills `out`)."""
        import torch
        dev = logp.device
        if stream is None:
            stream = torch.cuda.current_stream(dev)
        T = batch.total_tokens
        if out is None:
            out = {"loss": torch.empty(1, dtype=torch.float32, device=dev)}
            if grad:
                out["grad_logp"] = torch.empty(max(T, 4), dtype=torch.float32, device=dev)[:T]
            if stats:
                out["stats"] = torch.empty(LOSS_NSTATS, dtype=torch.float64, device=dev)
        lp = LossParams(float(clip_low), float(clip_high), float(beta_kl), float(lambda_eff), LOSS_FORMS[form],
                        LOSS_NORMS[norm])

        def pt(t):
            return None if t is None or t.numel() == 0 else t.data_ptr()

        li = LossInputs(pt(logp), pt(old_logp), pt(ref_logp), pt(edge_adv), pt(edge_cor), pt(edge_eff),
                        pt(edge_eff_mask))
        lo = LossOutputs(pt(out["loss"]), pt(out.get("grad_logp")), pt(out.get("stats")))
        cb = batch.c_struct()
        code = self._lib.gpo_token_loss(self._h, ctypes.byref(cb), plan.data_ptr(), ctypes.byref(lp),
                                        ctypes.byref(li), ctypes.byref(lo), ctypes.c_void_p(stream.cuda_stream))
        if code != GPO_OK:
            raise GraphPOError(code, self.last_error())
        return out

    def enable_timing(self, on: bool = True) -> None:
        code = self._lib.gpo_enable_timing(self._h, int(on))
        if code != GPO_OK:
            raise GraphPOError(code, self.last_error())

    def stage_times(self) -> dict:
        """{stage name: device ms} of the last call (timing must be enabled)."""
        cap = 16
        ms = (ctypes.c_float * cap)()
        names = (ctypes.c_char_p * cap)()
        n = ctypes.c_int()
        code = self._lib.gpo_stage_times(self._h, ms, names, cap, ctypes.byref(n))
        if code != GPO_OK:
            raise GraphPOError(code, self.last_error())
        return {names[i].decode(): float(ms[i]) for i in range(n.value)}

    def check(self, stream=None) -> None:
        import torch
        if stream is None:
            stream = torch.cuda.current_stream()
        code = self._lib.gpo_sync_status(self._h, ctypes.c_void_p(stream.cuda_stream))
        if code != GPO_OK:
            raise GraphPOError(code, self.last_error())

    def compute_host(self, host_batch: Batch, out=None, stream=None, chunk_bytes=0) -> "torch.Tensor":
        """End-to-end call on HOST tensors (pinned for asynchronous copies) through
        gpo_compute_host: the library uploads the batch into device staging buffers (kept
        here between calls of the same shape), runs the path over chunks of groups with the
        uploads of later chunks overlapping the work on earlier ones, and copies the
        per-token advantages back into `out` (a pinned float32 tensor of total_tokens
        elements, allocated if None).  chunk_bytes: embedding bytes per pipeline stage (0:
        the library's default).  Waits for the result and raises on a device-side error."""
        import torch
        dev = torch.device("cuda", torch.cuda.current_device())
        main = torch.cuda.current_stream(dev) if stream is None else stream
        names = ("group_rollout_off", "rollout_step_off", "step_len", "rollout_token_off", "emb", "reward",
                 "root_emb", "parent", "group_state_off", "group_token_off")
        host = [getattr(host_batch, n) for n in names]
        key = (dev, tuple(None if t is None else (tuple(t.shape), t.dtype) for t in host))
        if getattr(self, "_stage_key", None) != key:
            self._staged = [None if t is None else torch.empty(t.shape, dtype=t.dtype, device=dev) for t in host]
            self._stage_key = key
            self._stage_out = None
        if out is None:
            out = torch.empty(host_batch.total_tokens, dtype=torch.float32, pin_memory=True)
        db = Batch(*self._staged[:6], host_batch.total_tokens, host_batch.max_states_per_group, *self._staged[6:])
        if self._stage_out is None:
            self._stage_out = self.alloc_outputs(db)
        ws = self.workspace(db)
        hb, cb, co = host_batch.c_struct(), db.c_struct(), _c_outputs(self._stage_out)
        code = self._lib.gpo_compute_host(self._h, ctypes.byref(hb), ctypes.byref(cb), ctypes.byref(co),
                                          out.data_ptr() if out.numel() else None, int(chunk_bytes), ws.data_ptr(),
                                          ws.numel(), ctypes.c_void_p(main.cuda_stream))
        if code != GPO_OK:
            raise GraphPOError(code, self.last_error())
        self.check(main)
        return out
