"""The C-ABI library builds for sm_103a, loads, and exports every entry point
that include/lodestar.h declares; host-side argument checks answer without a
GPU (no compute call is made here)."""
import ctypes as C
import os
import re

import pytest

from paper_2606_00946_gb300 import build as B
from paper_2606_00946_gb300 import lodestar as L

INCLUDE = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")
HEADER = os.path.join(INCLUDE, "lodestar.h")
HEADERS = [HEADER, os.path.join(INCLUDE, "lodestar_probe.h")]


def declared_functions():
    src = "\n".join(open(h).read() for h in HEADERS)
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[A-Za-z_][\w\s\*]*?\b(ls_\w+)\s*\(", src, flags=re.M)))


@pytest.fixture(scope="module")
def lib():
    B.build()
    return L.lib()


def test_header_declares_the_boundary():
    names = declared_functions()
    for must in ("ls_create", "ls_destroy", "ls_snapshot_update", "ls_route_batch", "ls_train_step",
                 "ls_publish", "ls_log_samples", "ls_hash_blocks"):
        assert must in names
    assert set(names) == set(L._SIGS), "binding and header disagree"


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def _cfg(**kw):
    base = dict(widths=[16, 64, 64, 1], d_inst=10, d_req=0, dtype="f32")
    base.update(kw)
    return L.make_config(**base)


def test_param_count_and_config_validation(lib):
    assert L.ls_param_count(_cfg()) == 16 * 64 + 64 + 64 * 64 + 64 + 64 + 1
    bad = [
        _cfg(widths=[17, 64, 1]),                   # widths[0] != 6 + d_inst + d_req
        _cfg(widths=[16, 64, 2]),                   # output width must be 1
        _cfg(max_load=1.0),
        _cfg(max_load=0.0),
        _cfg(max_instances=0),
        _cfg(ring_capacity=0),
    ]
    for c in bad:
        assert L.ls_param_count(c) == L.LS_ERR_ARG
        rc, h = L.ls_create(c)
        assert rc == L.LS_ERR_ARG and not h.value
        assert L.last_error()
    c = _cfg()
    c.n_layers = 0
    assert L.ls_param_count(c) == L.LS_ERR_ARG


def test_null_arguments_rejected_on_host(lib):
    assert lib.ls_create(None, None) == L.LS_ERR_ARG
    assert lib.ls_route_batch(None, 1, None, None, None, None, None, None, None, None, None) == L.LS_ERR_ARG
    assert lib.ls_train_step(None, 1, None, 0, C.c_float(1e-3), None, None) == L.LS_ERR_ARG
    assert lib.ls_publish(None, None) == L.LS_ERR_ARG
    assert lib.ls_sync_status(None) == L.LS_ERR_ARG
    lib.ls_destroy(None)


def test_tensor_core_scorer_rejected_for_unsupported_predictors(lib):
    # fp32 predictor, and a bf16 predictor whose hidden width is not a multiple of 64
    for c in (_cfg(scorer="tensor_cores"),
              L.make_config([16, 48, 1], 10, 0, "bf16", scorer="tensor_cores")):
        rc, h = L.ls_create(c)
        assert rc == L.LS_ERR_ARG and not h.value
        assert "tensor-core" in L.last_error()
    bad = _cfg()
    bad.scorer = 7
    assert L.ls_param_count(bad) == L.LS_ERR_ARG


def test_prefix_index_mode_needs_at_most_512_instances(lib):
    c = _cfg(max_instances=600, prefix_mode="index")
    rc, h = L.ls_create(c)
    assert rc == L.LS_ERR_ARG and "512" in L.last_error()


@pytest.mark.parametrize("struct", [L.ls_config, L.ls_info, L.ls_guards])
def test_struct_layouts_match_the_header(struct, tmp_path):
    # sizeof and every field offset as gcc lays out the header's struct, against
    # the ctypes binding (a field added on one side only would shift the rest)
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    name = struct.__name__
    lines = [f'printf("size %zu\\n", sizeof({name}));']
    for f, _ in struct._fields_:
        lines.append(f'printf("{f} %zu\\n", offsetof({name}, {f}));')
    src = tmp_path / "layout.c"
    src.write_text('#include <stddef.h>\n#include <stdio.h>\n#include "lodestar.h"\nint main(void) {\n  '
                   + "\n  ".join(lines) + "\n  return 0;\n}\n")
    exe = tmp_path / "layout"
    subprocess.run([cc, "-I", os.path.dirname(HEADER), str(src), "-o", str(exe)], check=True)
    got = dict(line.split() for line in subprocess.run([str(exe)], capture_output=True, text=True,
                                                          check=True).stdout.splitlines())
    assert int(got["size"]) == C.sizeof(struct)
    for f, _ in struct._fields_:
        assert int(got[f]) == getattr(struct, f).offset, f
