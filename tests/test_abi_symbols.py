"""The C-ABI library loads and exports every entry point include/bom.h declares
(no compute: this runs without a GPU)."""
import os
import re

import pytest

from paper_2609_36738_gb300 import bom as B
from paper_2609_36738_gb300 import inputs as I

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "bom.h")


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    names = re.findall(r"^\s*(?:[A-Za-z_][\w\s\*]*?)\b(bom_\w+)\s*\(", src, flags=re.M)
    return sorted(set(names))


@pytest.fixture(scope="module")
def built():
    from paper_2609_36738_gb300 import build
    build.build()
    return B.lib()


def test_header_lists_the_expected_entry_points():
    assert declared_functions() == sorted(B.EXPORTED)


def test_library_exports_every_declared_symbol(built):
    for name in declared_functions():
        assert hasattr(built, name), name


def test_status_strings(built):
    for code in range(B.BOM_ESHARD + 1):
        assert B.status_string(code).startswith("BOM_")
    assert B.status_string(B.BOM_ESHARD + 1) == "unknown bom_status"


def test_param_layout_matches_workload_description(built):
    for wl in I.WORKLOADS.values():
        cfg = B.config_for(wl)
        shapes = wl.param_shapes()
        assert B.bom_param_count(cfg) == len(shapes)
        for i, (_, shape, _) in enumerate(shapes):
            assert B.bom_param_shape(cfg, i) == tuple(shape)


def test_workspace_sizes_and_config_checks(built):
    cfg = B.config_for(I.LM_MLP_BF16)
    ws = B.bom_workspace_bytes(cfg)
    # activations of two SwiGLU layers + logits dominate: a few GB, well inside HBM
    assert 2e9 < ws < 20e9
    bad = B.config_for(I.LM_HEAD_SMALL)
    bad.beta1 = 1.0
    assert B.bom_workspace_bytes(bad) == -1
    # a SwiGLU layer needs the bf16 tensor-core path
    f32 = B.make_config(16, 64, 10, [(B.BOM_LAYER_SWIGLU, 0, 64, 128)], False, B.BOM_F32)
    assert B.bom_workspace_bytes(f32) == -1
    # bf16 widths must be multiples of 8 (16-byte TMA row pitch)
    odd = B.make_config(16, 60, 10, [], False, B.BOM_BF16)
    assert B.bom_workspace_bytes(odd) == -1
