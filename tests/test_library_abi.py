"""The C-ABI library builds, loads and exports every entry point include/lacache.h declares (CPU only: no
compute calls are made here)."""
import ctypes
import os
import re
import subprocess

import pytest

from paper_2608_01718_gb300 import build, lacache

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "lacache.h")


@pytest.fixture(scope="module")
def lib():
    build.build()
    return lacache.load()


def declared_functions():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:lacache_status|const char\*|size_t)\s+(lacache_\w+)\s*\(", text, re.M)))


def test_header_is_strict_c99(tmp_path):
    src = tmp_path / "uses_header.c"
    src.write_text('#include "lacache.h"\nint main(void) { return lacache_status_string(LACACHE_OK) == 0; }\n')
    res = subprocess.run(["gcc", "-std=c99", "-Wall", "-Wextra", "-Wpedantic", "-Werror", "-fsyntax-only",
                          "-I", os.path.dirname(HEADER), str(src)], capture_output=True, text=True)
    assert res.returncode == 0, res.stderr


def test_c_client_compiles_against_the_header(tmp_path):
    client = os.path.join(os.path.dirname(os.path.abspath(__file__)), "c_client", "lookup_client.c")
    cuda_inc = os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "include")
    res = subprocess.run(["gcc", "-std=c99", "-Wall", "-Wextra", "-Werror", "-fsyntax-only", "-I",
                          os.path.dirname(HEADER), "-I", cuda_inc, client], capture_output=True, text=True)
    assert res.returncode == 0, res.stderr


def test_header_declares_the_binding_names():
    assert declared_functions() == sorted(lacache.EXPORTS)


def test_every_declared_symbol_is_exported(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name
        assert ctypes.cast(getattr(lib, name), ctypes.c_void_p).value


def test_status_strings(lib):
    assert lacache.status_string(lacache.LACACHE_OK) == "ok"
    assert lacache.status_string(lacache.LACACHE_ERR_IO) == "i/o error"
    assert lacache.status_string(lacache.LACACHE_ERR_CAPACITY) == "capacity exceeded"
    assert lacache.status_string(99) == "unknown status"


def test_struct_layouts_match_the_header():
    # lacache_config: 2 x int32, int64, 2 x float, 6 x int32 = 48 bytes; lacache_result: 13 pointers;
    # lacache_shard_result: 8 pointers and an int64;
    # lacache_ensemble: int32 + 8 int32 + 8 float
    assert ctypes.sizeof(lacache.lacache_config) == 48
    assert lacache.lacache_config.capacity.offset == 8
    assert ctypes.sizeof(lacache.lacache_result) == 104
    assert ctypes.sizeof(lacache.lacache_shard_result) == 72
    assert ctypes.sizeof(lacache.lacache_stats) == 56
    assert ctypes.sizeof(lacache.lacache_ensemble) == 68


def test_invalid_ensembles_are_rejected_before_touching_a_device(lib):
    cfg = lacache.make_config(64, 8, 1024, 0.9, 0.8, 8, max_batch=16)
    h = ctypes.c_void_p(1)
    for dims, taus, status in [((), (), lacache.LACACHE_ERR_INVALID_ARG),
                               ((64, 12), (0.7, 0.7), lacache.LACACHE_ERR_UNSUPPORTED),
                               ((64, 0), (0.7, 0.7), lacache.LACACHE_ERR_INVALID_ARG),
                               ((64, 64), (0.7, float("nan")), lacache.LACACHE_ERR_INVALID_ARG),
                               ((64,) * 9, (0.7,) * 9, lacache.LACACHE_ERR_INVALID_ARG)]:
        ens = lacache.lacache_ensemble()
        ens.m = len(dims)
        for i, (d, t) in enumerate(zip(dims[:8], taus[:8])):
            ens.dims[i], ens.tau_a[i] = d, t
        assert lib.lacache_create_ensemble(ctypes.byref(cfg), ctypes.byref(ens), ctypes.byref(h)) == status
        assert h.value is None


def test_null_arguments_are_rejected_without_a_device(lib):
    h = ctypes.c_void_p()
    assert lib.lacache_create(None, ctypes.byref(h)) == lacache.LACACHE_ERR_INVALID_ARG
    assert lib.lacache_create(ctypes.byref(lacache.make_config(64, 4, 16, .9, .8, 4, max_batch=8)), None) == \
        lacache.LACACHE_ERR_INVALID_ARG
    assert lib.lacache_destroy(None) == lacache.LACACHE_OK
    assert lib.lacache_sync(None) == lacache.LACACHE_ERR_INVALID_ARG
    n = ctypes.c_int64()
    assert lib.lacache_size(None, ctypes.byref(n)) == lacache.LACACHE_ERR_INVALID_ARG


@pytest.mark.parametrize("field,value,status", [
    ("d", 12, lacache.LACACHE_ERR_UNSUPPORTED), ("d", 0, lacache.LACACHE_ERR_INVALID_ARG),
    ("top_c", 33, lacache.LACACHE_ERR_UNSUPPORTED), ("k", 0, lacache.LACACHE_ERR_INVALID_ARG),
    ("check_mode", 7, lacache.LACACHE_ERR_INVALID_ARG), ("token_match_min", 9, lacache.LACACHE_ERR_INVALID_ARG),
    ("tau_c", float("nan"), lacache.LACACHE_ERR_INVALID_ARG), ("max_batch", 0, lacache.LACACHE_ERR_INVALID_ARG),
])
def test_invalid_configs_are_rejected_before_touching_a_device(lib, field, value, status):
    cfg = lacache.make_config(64, 8, 1024, 0.9, 0.8, 8, max_batch=16)
    setattr(cfg, field, value)
    h = ctypes.c_void_p(1)
    assert lib.lacache_create(ctypes.byref(cfg), ctypes.byref(h)) == status
    assert h.value is None


def test_load_rejects_what_is_not_a_saved_cache_before_touching_a_device(lib, tmp_path):
    h = ctypes.c_void_p(1)
    missing = str(tmp_path / "missing.lacache").encode()
    assert lib.lacache_load(missing, 0, 0, ctypes.byref(h)) == lacache.LACACHE_ERR_IO and h.value is None
    bad = tmp_path / "bad.lacache"
    bad.write_bytes(b"NOTACACHE" + bytes(200))
    assert lib.lacache_load(str(bad).encode(), 0, 0, ctypes.byref(h)) == lacache.LACACHE_ERR_IO
    short = tmp_path / "short.lacache"
    short.write_bytes(b"LACACHE1" + bytes(10))          # magic, then a truncated header
    assert lib.lacache_load(str(short).encode(), 0, 0, ctypes.byref(h)) == lacache.LACACHE_ERR_IO
    assert lib.lacache_load(str(short).encode(), 0, -1, ctypes.byref(h)) == lacache.LACACHE_ERR_INVALID_ARG
    assert lib.lacache_save(None, b"x") == lacache.LACACHE_ERR_INVALID_ARG


def test_a_missing_library_raises_instead_of_falling_back(monkeypatch, tmp_path):
    # the product path has no CPU route: without liblacache.so every binding call fails loudly
    monkeypatch.setattr(lacache, "LIB_PATH", str(tmp_path / "liblacache.so"))
    monkeypatch.setattr(lacache, "_lib", None)
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        lacache.load()
    with pytest.raises(RuntimeError, match="is missing"):
        lacache.lacache_create(lacache.make_config(64, 8, 1024, 0.9, 0.8, 8, max_batch=16))
    with pytest.raises(RuntimeError, match="is missing"):
        lacache.status_string(lacache.LACACHE_OK)


def test_candidate_packing_orders_scores_then_ids(tmp_path):
    """The stage-1 kernels' packed (score, id) candidates, compiled for the host from the same header: their
    unsigned order is (score descending, id ascending), and -0.0 ties with +0.0."""
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    src = os.path.join(root, "tests", "c_client", "pack_order_check.cu")
    exe = tmp_path / "pack_order_check"
    res = subprocess.run([build.nvcc(), "-std=c++17", "-I", os.path.join(root, "include"), "-I", build.CSRC,
                          src, "-o", str(exe)], capture_output=True, text=True)
    assert res.returncode == 0, res.stdout + res.stderr
    run = subprocess.run([str(exe)], capture_output=True, text=True)
    assert run.returncode == 0, run.stderr
