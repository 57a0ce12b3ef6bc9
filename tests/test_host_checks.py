"""Host-side checks of the C ABI that need no GPU: gpo_workspace_size (no context) and
gpo_loss_plan_size read only a batch's sizes and the nullness and alignment of its
pointers, so every validation code they share with gpo_compute is reachable on the CPU.
The batches here live in host memory; nothing dereferences their pointers."""
import ctypes

import pytest

from paper_2606_18954_gb300 import binding as B
from paper_2606_18954_gb300 import workloads as W

OK, INVALID, SHAPE, UNSUPPORTED = 0, 1, 2, 5


@pytest.fixture(scope="module")
def lib():
    from paper_2606_18954_gb300 import build
    build()
    return B.load()


def _chain(groups=4, dtype=None):
    spec = W.CONFIGS["tiny"].scaled(groups=groups)
    if dtype is not None:
        spec = spec.scaled(dtype=dtype)
    return B.Batch.from_arrays(W.make_batch(spec, seed=11), device="cpu")


def _tree(groups=3):
    spec = W.TREE_CONFIGS["tree"].scaled(groups=groups, d=64)
    return B.Batch.from_arrays(W.make_tree_batch(spec, seed=12), device="cpu")


def _status(lib, cb):
    n = ctypes.c_size_t(0)
    return lib.gpo_workspace_size(None, ctypes.byref(cb), ctypes.byref(n)), n.value


def test_workspace_size_without_context(lib):
    small, large = _chain(4), _chain(16)
    a, b = B.workspace_size(small), B.workspace_size(large)
    assert a > 0 and a % 256 == 0 and b % 256 == 0
    assert b > a  # grows with the states and groups
    t = B.workspace_size(_tree())
    assert t > 0 and t % 256 == 0


def test_workspace_size_of_an_empty_batch(lib):
    cb = _chain(1).c_struct()
    cb.num_groups = cb.num_rollouts = cb.num_states = 0
    cb.total_tokens = 0
    cb.max_states_per_group = 0
    code, n = _status(lib, cb)
    assert code == OK and n > 0


def _stride_reaching(elements, rows):
    """The smallest fp32 row stride of 16-byte rows with rows x stride >= elements."""
    s = -(-elements // rows)
    return (s + 3) // 4 * 4


def test_stride_helper():
    s = _stride_reaching(1 << 40, 96)
    assert s * 96 >= 1 << 40 and (s - 4) * 96 < 1 << 40 and (s * 4) % 16 == 0 and s < 1 << 40


CHAIN_CASES = {
    "negative groups": (lambda c: setattr(c, "num_groups", -1), INVALID),
    "negative tokens": (lambda c: setattr(c, "total_tokens", -5), INVALID),
    "d = 0": (lambda c: setattr(c, "d", 0), INVALID),
    "unknown dtype": (lambda c: setattr(c, "emb_dtype", 7), INVALID),
    "group above the maximum": (lambda c: setattr(c, "max_states_per_group", 4097), UNSUPPORTED),
    "no group size with states": (lambda c: setattr(c, "max_states_per_group", 0), INVALID),
    "more rollouts than states": (lambda c: setattr(c, "num_rollouts", c.num_states + 1), SHAPE),
    "row stride below d": (lambda c: setattr(c, "emb_row_stride", c.d - 1), INVALID),
    "row bytes not a multiple of 16": (lambda c: (setattr(c, "d", 3), setattr(c, "emb_row_stride", 3)), UNSUPPORTED),
    "embeddings misaligned": (lambda c: setattr(c, "emb", c.emb + 4), UNSUPPORTED),
    "root embeddings misaligned": (lambda c: setattr(c, "root_emb", c.emb + 8), UNSUPPORTED),
    # a stride whose product with the state count would overflow int64
    "row stride too large": (lambda c: setattr(c, "emb_row_stride", 1 << 60), UNSUPPORTED),
    "embedding matrix too large": (lambda c: setattr(c, "emb_row_stride", _stride_reaching(1 << 40, c.num_states)),
                                   UNSUPPORTED),
    "tree offsets without parent": (lambda c: setattr(c, "group_state_off", c.rollout_step_off), INVALID),
    "rollout_step_off NULL": (lambda c: setattr(c, "rollout_step_off", None), INVALID),
    "rollout_token_off NULL": (lambda c: setattr(c, "rollout_token_off", None), INVALID),
    "group_rollout_off NULL": (lambda c: setattr(c, "group_rollout_off", None), INVALID),
    "step_len NULL": (lambda c: setattr(c, "step_len", None), INVALID),
    "emb NULL": (lambda c: setattr(c, "emb", None), INVALID),
    "reward NULL": (lambda c: setattr(c, "reward", None), INVALID),
}


@pytest.mark.parametrize("name", sorted(CHAIN_CASES))
def test_chain_batch_checks(lib, name):
    cb = _chain(2).c_struct()
    assert _status(lib, cb)[0] == OK
    mutate, want = CHAIN_CASES[name]
    mutate(cb)
    assert _status(lib, cb)[0] == want


TREE_CASES = {
    "group_state_off NULL": (lambda c: setattr(c, "group_state_off", None), INVALID),
    "group_token_off NULL": (lambda c: setattr(c, "group_token_off", None), INVALID),
    "group_rollout_off NULL": (lambda c: setattr(c, "group_rollout_off", None), INVALID),
}


@pytest.mark.parametrize("name", sorted(TREE_CASES))
def test_tree_batch_checks(lib, name):
    cb = _tree().c_struct()
    assert cb.rollout_step_off is None and cb.rollout_token_off is None
    assert _status(lib, cb)[0] == OK  # the chain-only offsets are not read
    mutate, want = TREE_CASES[name]
    mutate(cb)
    assert _status(lib, cb)[0] == want


def test_fp32_rows_of_16_bytes_are_accepted(lib):
    cb = _chain(2).c_struct()
    cb.d = 4
    cb.emb_row_stride = 4
    assert _status(lib, cb)[0] == OK
    cb.emb_dtype = B.EMB_BF16  # 8 bytes a row
    assert _status(lib, cb)[0] == UNSUPPORTED


def test_workspace_size_needs_an_output_pointer(lib):
    cb = _chain(2).c_struct()
    assert lib.gpo_workspace_size(None, ctypes.byref(cb), None) == INVALID
    assert lib.gpo_workspace_size(None, None, None) == INVALID


def test_binding_raises_the_status(lib):
    b = _chain(2)
    cb = b.c_struct()
    cb.max_states_per_group = 5000
    with pytest.raises(B.GraphPOError) as e:
        B.workspace_size(cb)
    assert e.value.code == UNSUPPORTED


def test_loss_plan_size(lib):
    small, large = _chain(4), _chain(16)
    a, b = B.loss_plan_size(small), B.loss_plan_size(large)
    assert a > 0 and a % 256 == 0 and b > a
    assert B.loss_plan_size(_tree()) % 256 == 0
    cb = small.c_struct()
    cb.total_tokens = -1
    n = ctypes.c_size_t()
    assert lib.gpo_loss_plan_size(ctypes.byref(cb), ctypes.byref(n)) == INVALID
    assert lib.gpo_loss_plan_size(None, ctypes.byref(n)) == INVALID
    cb = small.c_struct()
    cb.num_groups = cb.num_rollouts = cb.num_states = 0
    cb.total_tokens = 0
    assert lib.gpo_loss_plan_size(ctypes.byref(cb), ctypes.byref(n)) == OK and n.value > 0
