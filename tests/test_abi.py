"""C-ABI boundary checks that need no GPU: the library builds for sm_103a, loads,
exports every function include/graphpo.h declares, and the binding's structs
match the header's field lists."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "graphpo.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2606_18954_gb300 import build, load
    build()
    return load()


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(gpo_[a-z_]+)\s*\(", src)))


def struct_fields(name):
    src = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    m = re.search(r"typedef struct \{([^{}]*)\}\s*" + name + ";", src)
    body = m.group(1)
    fields = []
    for decl in body.split(";"):
        decl = decl.strip()
        if not decl:
            continue
        for part in decl.split(","):
            ident = re.findall(r"\*?\s*([A-Za-z_][A-Za-z_0-9]*)\s*$", part.strip())
            fields.append(ident[0])
    return fields


def test_exports_every_declared_function(lib):
    names = declared_functions()
    assert len(names) >= 8
    so = lib._name
    out = subprocess.run(["nm", "-D", "--defined-only", so], capture_output=True, text=True).stdout
    exported = set(re.findall(r"\bT (gpo_[a-z_]+)", out))
    for n in names:
        assert n in exported, n
        assert hasattr(lib, n)


def test_binding_structs_match_header():
    from paper_2606_18954_gb300 import binding as B
    assert [f for f, _ in B.Params._fields_] == struct_fields("gpo_params")
    assert [f for f, _ in B.CBatch._fields_] == struct_fields("gpo_batch")
    assert [f for f, _ in B.COutputs._fields_] == struct_fields("gpo_outputs")
    assert [f for f, _ in B.LossParams._fields_] == struct_fields("gpo_loss_params")
    assert [f for f, _ in B.LossInputs._fields_] == struct_fields("gpo_loss_inputs")
    assert [f for f, _ in B.LossOutputs._fields_] == struct_fields("gpo_loss_outputs")
    assert sorted(B.EXPORTS) == declared_functions()


def test_status_strings_and_version(lib):
    assert lib.gpo_version().startswith(b"graphpo-gb300")
    for code in range(10):
        assert lib.gpo_status_string(code)
    assert lib.gpo_status_string(123) == b"unknown status"


def test_argument_checks_without_device(lib):
    from paper_2606_18954_gb300 import binding as B
    h = ctypes.c_void_p()
    bad = B.Params(0.92, 1.5, 1.0, 1e-6, 1, 0, 0)   # w outside [0, 1]
    assert lib.gpo_create(ctypes.byref(h), ctypes.byref(bad)) == 1
    bad = B.Params(0.92, 0.7, -1.0, 1e-6, 1, 0, 0)  # negative lambda
    assert lib.gpo_create(ctypes.byref(h), ctypes.byref(bad)) == 1
    bad = B.Params(0.0, 0.7, 1.0, 1e-6, 1, 0, 0)    # kappa must be positive
    assert lib.gpo_create(ctypes.byref(h), ctypes.byref(bad)) == 1
    assert lib.gpo_create(None, None) == 1
    assert lib.gpo_sync_status(None, None) == 1
    assert lib.gpo_compute(None, None, None, None, 0, None) == 1
    assert lib.gpo_last_error(None) == b"no context"


def test_product_never_imports_the_oracle():
    """The product package must not import, load or run anything under oracle/."""
    pkg = os.path.join(ROOT, "paper_2606_18954_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h")):
                txt = open(os.path.join(dirpath, f)).read()
                assert "import oracle" not in txt and "liboracle" not in txt and "oracle.c" not in txt, f


C_CLIENT = r"""
#include <stdio.h>
#include <string.h>
#include "graphpo.h"

int main(void) {
  /* a plain C99 client: the header needs no CUDA or C++ types; host-only calls work
     without a device */
  gpo_batch b;
  size_t bytes = 0;
  int32_t go[1] = {0}, so[1] = {0};
  int64_t to[1] = {0};
  memset(&b, 0, sizeof b);  /* an empty batch: no groups, rollouts, states or tokens */
  b.d = 8;
  b.emb_row_stride = 8;
  b.group_rollout_off = go;  /* the offset arrays (G + 1, R + 1 entries) are required */
  b.rollout_step_off = so;
  b.rollout_token_off = to;
  if (gpo_workspace_size(NULL, &b, &bytes) != GPO_OK || bytes == 0) return 1;
  b.num_groups = -1;
  if (gpo_workspace_size(NULL, &b, &bytes) != GPO_ERR_INVALID_ARG) return 2;
  if (strncmp(gpo_version(), "graphpo-gb300", 13) != 0) return 3;
  printf("%s|%s|%zu\n", gpo_version(), gpo_status_string(GPO_ERR_SHAPE), bytes);
  return 0;
}
"""


def test_header_is_plain_c_and_links(lib, tmp_path):
    """include/graphpo.h compiles as C99 with warnings as errors, and a C program links
    against the library and calls its host-only entry points."""
    src = tmp_path / "client.c"
    src.write_text(C_CLIENT)
    exe = tmp_path / "client"
    so = lib._name
    subprocess.check_call(["gcc", "-std=c99", "-Wall", "-Wextra", "-Werror", "-pedantic", "-I",
                           os.path.join(ROOT, "include"), str(src), "-o", str(exe), so,
                           "-Wl,-rpath," + os.path.dirname(so)])
    out = subprocess.run([str(exe)], capture_output=True, text=True)
    assert out.returncode == 0, out
    assert out.stdout.startswith("graphpo-gb300") and "inconsistent offsets" in out.stdout


def test_debug_build_compiles_and_loads():
    """The debug build (GPO_DEBUG: index checks in every kernel, GPO_ERR_BOUNDS) compiles for
    sm_103a, loads, says so in gpo_version and names the extra status."""
    from paper_2606_18954_gb300 import buildlib
    path = buildlib.build(debug=True)
    assert path == buildlib.DEBUG_LIB and path != buildlib.LIB
    L = ctypes.CDLL(path)
    L.gpo_version.restype = ctypes.c_char_p
    L.gpo_status_string.restype = ctypes.c_char_p
    L.gpo_status_string.argtypes = [ctypes.c_int]
    assert b"GPO_DEBUG" in L.gpo_version()
    assert b"debug build" in L.gpo_status_string(9)
