"""The C-ABI library loads and exports every entry point declared in include/netkv.h.

No compute calls: only entry points that fail on host-side validation before
touching a GPU are called here."""
import ctypes as C
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "netkv.h")


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2606_03910_gb300 import netkv
    return netkv


def declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(netkv_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared()
    for n in ("netkv_topology_create", "netkv_topology_destroy", "netkv_topology_query",
              "netkv_oracle_build", "netkv_cache_build", "netkv_prefix_match",
              "netkv_schedule_streams", "netkv_version"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    so = C.CDLL(lib.LIB_PATH)
    for name in declared():
        assert hasattr(so, name), f"{name} not exported"
    assert set(lib.EXPORTS) <= set(declared())


def test_every_entry_point_declares_its_argument_types(lib):
    """Without argtypes ctypes passes Python ints as 32-bit C ints, truncating device
    pointers; every entry point of the binding must declare its argument types."""
    for name in lib.EXPORTS:
        if name == "netkv_version":
            continue
        assert getattr(lib._lib, name).argtypes is not None, name


def test_version_and_host_validation(lib):
    assert lib.netkv_version() >= 1
    import numpy as np
    with pytest.raises(lib.NetKVError) as e:
        lib.netkv_topology_create((2, 0, 2, 2), np.zeros(0, np.uint8), (1, 1, 1, 1), (0, 0, 0, 0), 8)
    assert e.value.code == lib.NETKV_EINVAL
    so = lib._lib
    assert so.netkv_oracle_build(None, None, 1, 1.0, None, None, None, None) == lib.NETKV_EINVAL
    assert so.netkv_cache_build(None, 1, 1, 4, None, None, None, None) == lib.NETKV_EINVAL
    # per (set, group of 64 decodes): slots (16 B), run keys (8 B) and run masks (1, 2, 4 or
    # 8 B by pool size) per position, padded to 256 bytes
    assert so.netkv_cache_index_bytes(2, 65, 4) == 2 * 2 * (16 + 8 + 8) * 16
    assert so.netkv_cache_index_bytes(3, 8, 10) == 3 * (16 + 8 + 1) * 1024
    assert so.netkv_cache_index_bytes(1, 16, 10) == (16 + 8 + 2) * 1024
    assert so.netkv_cache_index_bytes(1, 20, 10) == (16 + 8 + 4) * 1024
    assert so.netkv_cache_index_bytes(1, 8, 1) == 256
    assert so.netkv_prefix_match(None, 1, 4, 1, None, None, 1, None, None, 0, None, None, None) == lib.NETKV_EINVAL
    assert so.netkv_prefix_match_workspace_size(0) == 0
    assert so.netkv_schedule_streams(None, 1, None, 0, None, None, None, None, None, 0, None, None,
                                     None, None, None, None, None, None, 0, None,
                                     None) == lib.NETKV_EINVAL
    assert so.netkv_schedule_workspace_size(10, 8) == 512
    assert so.netkv_schedule_streams_inflight(None, 1, None, 0, None, None, None, None, None,
                                              None, 0, None, None, 16, None, None, None, None,
                                              None, None, None, 0, None, None) == lib.NETKV_EINVAL
    assert so.netkv_schedule_inflight_workspace_size(10, 8) == 1024
    assert so.netkv_topology_destroy(None) == lib.NETKV_EINVAL


def test_load_model_layout(lib):
    """netkv_load_model: two floats, two int32, two int64 in 32 bytes."""
    M = lib.LoadModel
    assert C.sizeof(M) == 32
    assert [getattr(M, f).offset for f, _ in M._fields_] == [0, 4, 8, 12, 16, 24]


def test_weights_layout(lib):
    assert lib.WEIGHTS_DTYPE.itemsize == 32
    assert [lib.WEIGHTS_DTYPE.fields[k][1] for k in lib.WEIGHTS_DTYPE.names] == [0, 4, 8, 12, 16, 24]


def test_product_path_does_not_import_the_oracle():
    """The library package and its binding never reference the oracle."""
    pkg = os.path.join(ROOT, "paper_2606_03910_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h")):
                src = open(os.path.join(dirpath, f)).read()
                assert "import oracle" not in src and "from oracle" not in src, f
                assert "netkv_oracle.cpp" not in src and "libnetkv_oracle" not in src, f
