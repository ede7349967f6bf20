"""CPU checks of the C ABI: the library builds for sm_103a, loads without a
GPU, exports every function include/oprag.h declares, and its host-side
argument checks reject bad calls before touching the device."""
import ctypes
import os
import re

import pytest

from paper_2608_08340_gb300 import _lib
from paper_2608_08340_gb300 import build as lib_build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    lib_build.build()
    return _lib.load()


def declared_functions():
    text = open(os.path.join(ROOT, "include", "oprag.h")).read()
    return sorted(set(re.findall(r"\b(oprag_\w+)\s*\(", text)))


def test_header_declares_the_expected_entry_points():
    names = declared_functions()
    for must in ("oprag_index_create", "oprag_upsert", "oprag_search", "oprag_hybrid_search",
                 "oprag_index_set_sparse", "oprag_last_error"):
        assert must in names


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_binding_covers_every_declared_symbol():
    assert sorted(_lib.SIGNATURES) == declared_functions()


def test_library_targets_sm103a_only():
    """Every nvcc command of the build (each compile and the link) names
    sm_103a as its only target."""
    assert lib_build.ARCH == "-gencode=arch=compute_103a,code=sm_103a"
    lib_build.build()
    if not os.path.exists(lib_build.COMMANDS_PATH):      # built before commands were recorded
        lib_build.build(force=True)
    lines = open(lib_build.COMMANDS_PATH).read().splitlines()
    srcs = lib_build.sources()
    assert len(lines) == len(srcs) + 1
    for line in lines:
        args = line.split()
        targets = [a for a in args if "arch=" in a or a.startswith("-arch") or "code=" in a]
        assert targets == [lib_build.ARCH], line
    for src, line in zip(srcs, lines):
        assert f" -c {src} " in line
    assert " -shared " in lines[-1]


def test_option_codes_match_header():
    text = open(os.path.join(ROOT, "include", "oprag.h")).read()
    for name, value in re.findall(r"#define (OPRAG_OPT_\w+) (\d+)", text):
        assert getattr(_lib, name) == int(value), name


def _err(lib):
    return lib.oprag_last_error().decode()


def test_null_and_shape_arguments_are_rejected_on_the_host(lib):
    h = ctypes.c_void_p()
    buf = (ctypes.c_float * 64)()
    # NULL output handle / NULL embeddings
    assert lib.oprag_index_create(None, buf, 8, 8, 1, 0, 0) == -1
    assert lib.oprag_index_create(ctypes.byref(h), None, 8, 8, 1, 0, 0) == -1
    assert "NULL" in _err(lib)
    # d not a multiple of 8, n = 0, unknown dtype, bf16 -> f32
    assert lib.oprag_index_create(ctypes.byref(h), buf, 8, 12, 1, 0, 0) == -1
    assert "multiple of 8" in _err(lib)
    assert lib.oprag_index_create(ctypes.byref(h), buf, 0, 8, 1, 0, 0) == -1
    assert lib.oprag_index_create(ctypes.byref(h), buf, 8, 8, 7, 0, 0) == -1
    assert lib.oprag_index_create(ctypes.byref(h), buf, 8, 8, 0, 1, 0) == -1
    assert h.value is None
    # calls on a NULL index
    assert lib.oprag_search(None, buf, 1, 1, buf, buf, None) == -1
    assert lib.oprag_hybrid_search(None, buf, 1, buf, buf, 0.5, 1, buf, buf, None) == -1
    assert lib.oprag_upsert(None, buf, buf, 1, 0, 0, None) == -1
    assert lib.oprag_index_check(None) == -1
    assert lib.oprag_index_info(None, None, None, None, None) == -1
    assert lib.oprag_index_last_path(None) == 0
    t = ctypes.c_int32()
    assert lib.oprag_index_last_tiles_per_cta(None, ctypes.byref(t)) == -1
    assert lib.oprag_index_last_launch(None, None, None, None) == -1
    plan = (ctypes.c_int64 * 13)()
    assert lib.oprag_plan_search(1000, 768, 16, 5, 148, 0, 0, 74, None) == -1
    assert lib.oprag_plan_search(1000, 768, 16, 5, 0, 0, 0, 74, plan) == -1
    assert lib.oprag_plan_search(1000, 768, 16, 5, 148, 0, 0, 74, plan) == 0
    lib.oprag_index_destroy(None)


def test_error_codes_match_header():
    text = open(os.path.join(ROOT, "include", "oprag.h")).read()
    codes = {int(v): k for k, v in re.findall(r"#define OPRAG_(?:ERR_)?(\w+) \((-\d+)\)", text)}
    for code, name in codes.items():
        assert _lib.ERRORS[code] == name
    assert int(re.search(r"#define OPRAG_K_MAX (\d+)", text).group(1)) == _lib.OPRAG_K_MAX
