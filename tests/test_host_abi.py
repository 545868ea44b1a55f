"""CPU tests of the C ABI: the library loads, exports exactly what
include/lamb.h declares, the host planner covers every element once, and
argument errors are reported before any device work.  No kernel runs here."""
import ctypes
import os
import re
import shutil
import subprocess

import numpy as np
import pytest

from conftest import ROOT, cuda_available
from paper_1904_00962_gb300 import binding as B
from paper_1904_00962_gb300 import build as build_mod

HEADER = os.path.join(ROOT, "include", "lamb.h")


@pytest.fixture(scope="module")
def lib():
    build_mod.build()
    return B.load()


def _declared():
    text = open(HEADER).read()
    return set(re.findall(r"^LAMB_API\s+[\w\s\*]+?\b(\w+)\s*\(", text, re.M))


def test_header_declares_the_boundary():
    names = _declared()
    for must in ("lamb_plan_create", "lamb_plan_bind", "lamb_step",
                 "lars_step", "lamb_plan_destroy"):
        assert must in names
    assert names == set(B.EXPORTED)


def test_library_exports_every_declared_symbol(lib):
    for name in _declared():
        assert hasattr(lib, name), name
    nm = shutil.which("nm")
    if nm:
        out = subprocess.run([nm, "-D", "--defined-only", B.LIB_PATH],
                             capture_output=True, text=True).stdout
        exported = {l.split()[-1] for l in out.splitlines()
                    if re.match(r"^[0-9a-f]+ T ", l)}
        assert exported == _declared()


def test_abi_version(lib):
    assert B.lamb_abi_version() == 1


def test_header_compiles_as_c():
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("gcc not available")
    inc = "/usr/local/cuda/include"
    src = '#include "lamb.h"\nint main(void){return LAMB_OK;}\n'
    res = subprocess.run([gcc, "-std=c99", "-Wall", "-Werror", "-fsyntax-only",
                          "-I", os.path.join(ROOT, "include"), "-I", inc,
                          "-x", "c", "-"], input=src, capture_output=True,
                         text=True)
    assert res.returncode == 0, res.stderr


def test_struct_sizes_match_ctypes():
    # lamb_hyper_t: 7 doubles + int32 + uint32 = 64 bytes
    assert ctypes.sizeof(B.lamb_hyper_t) == 64
    assert ctypes.sizeof(B.lamb_plan_options_t) == 8


# ---------------------------------------------------------------------------
# Host planner
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("chunk", [1024, 4096, 16384])
def test_chunk_table_covers_every_element_once(lib, chunk):
    rng = np.random.default_rng(chunk)
    sizes = [0, 1, 3, 1023, 1024, 1025, chunk, chunk + 1, 3 * chunk - 1,
             *rng.integers(1, 200000, 40).tolist(), 0]
    t, o, ln = B.lamb_layout_chunks(sizes, chunk)
    assert len(t) == sum((s + chunk - 1) // chunk for s in sizes)
    assert np.all(ln >= 1) and np.all(ln <= chunk)
    assert np.all(np.diff(t) >= 0)                   # tensor order
    for k, s in enumerate(sizes):
        sel = t == k
        if s == 0:
            assert not sel.any()
            continue
        offs, lens = o[sel], ln[sel]
        assert offs[0] == 0
        np.testing.assert_array_equal(offs[1:], offs[:-1] + lens[:-1])
        assert offs[-1] + lens[-1] == s
        assert np.all(lens[:-1] == chunk)            # only the last is ragged
        assert np.all(offs % 4 == 0)                 # vector-aligned starts


def test_chunk_table_default_chunk(lib):
    t, o, ln = B.lamb_layout_chunks([16384 * 3 + 5], 0)
    assert len(t) == 4 and ln[-1] == 5


def test_bert_large_chunk_count(lib):
    from paper_1904_00962_gb300.workloads import bert_large_layout
    L = bert_large_layout()
    t, o, ln = B.lamb_layout_chunks(L.sizes, 16384)
    assert int(ln.sum()) == L.n_params == 335141888
    assert len(set(t.tolist())) == 391


@pytest.mark.parametrize("sizes,chunk", [
    ([], 16384),                       # n = 0
    ([5, -1], 16384),                  # negative size
    ([5], 1000),                       # chunk not a multiple of 1024
    ([5], 1 << 25),                    # chunk too big
    ([1 << 61, 1 << 61, 1 << 61], 1 << 24),   # total > 2^62
    ([1 << 41], 1024),                 # more than 2^30 chunks
])
def test_planner_rejects_bad_input(lib, sizes, chunk):
    with pytest.raises(B.LambError) as ei:
        B.lamb_layout_chunks(sizes, chunk)
    assert ei.value.status == B.LAMB_ERR_INVALID_ARG
    assert B.lamb_last_error()


def test_planner_capacity_too_small(lib):
    sz = (ctypes.c_int64 * 1)(10000)
    n = ctypes.c_int32()
    t = (ctypes.c_int32 * 2)()
    o = (ctypes.c_int64 * 2)()
    ln = (ctypes.c_int32 * 2)()
    st = lib.lamb_layout_chunks(sz, 1, 1024, t, o, ln, 2, ctypes.byref(n))
    assert st == B.LAMB_ERR_INVALID_ARG and n.value == 10


# ---------------------------------------------------------------------------
# Argument validation before any device work
# ---------------------------------------------------------------------------

def test_create_validates_before_touching_the_device(lib):
    with pytest.raises(B.LambError) as ei:
        B.lamb_plan_create([10], grad_dtype=7)
    assert ei.value.status == B.LAMB_ERR_UNSUPPORTED_DTYPE
    with pytest.raises(B.LambError) as ei:
        B.lamb_plan_create([10], copy_dtype=B.LAMB_F32)
    assert ei.value.status == B.LAMB_ERR_UNSUPPORTED_DTYPE
    with pytest.raises(B.LambError) as ei:
        B.lamb_plan_create([])
    assert ei.value.status == B.LAMB_ERR_INVALID_ARG
    with pytest.raises(B.LambError) as ei:
        B.lamb_plan_create([10, -3])
    assert ei.value.status == B.LAMB_ERR_INVALID_ARG
    with pytest.raises(B.LambError) as ei:
        B.lamb_plan_create([10], chunk_elems=100)
    assert ei.value.status == B.LAMB_ERR_INVALID_ARG
    with pytest.raises(B.LambError) as ei:
        B.lamb_plan_create([10], device=-1)
    assert ei.value.status == B.LAMB_ERR_INVALID_ARG


@pytest.mark.skipif(cuda_available(), reason="checks the no-GPU error path")
def test_create_without_gpu_reports_cuda_error(lib):
    with pytest.raises(B.LambError) as ei:
        B.lamb_plan_create([10, 20])
    assert ei.value.status in (B.LAMB_ERR_CUDA, B.LAMB_ERR_OOM)
    assert "cuda" in str(ei.value).lower() or B.lamb_last_error()


def test_null_plan_is_rejected(lib):
    h = B.make_hyper()
    for fn in (lambda: B.lamb_step(0, h, 0, 0), lambda: B.lars_step(0, h, 0, 0),
               lambda: B.lamb_plan_bind(0, [1], [1], [1]),
               lambda: B.lamb_plan_query(0),
               lambda: B.lamb_plan_get_info(0),
               lambda: B.lamb_plan_copy_trust_ratios(0)):
        with pytest.raises(B.LambError) as ei:
            fn()
        assert ei.value.status == B.LAMB_ERR_INVALID_ARG
    B.lamb_plan_destroy(0)   # destroying NULL is a no-op


def test_last_error_is_thread_local(lib):
    import threading
    with pytest.raises(B.LambError):
        B.lamb_plan_create([], )
    msg_main = B.lamb_last_error()
    seen = {}

    def worker():
        seen["msg"] = B.lamb_last_error()
    th = threading.Thread(target=worker)
    th.start(); th.join()
    assert msg_main and seen["msg"] == ""


def test_product_path_fails_loudly_without_library(tmp_path):
    with pytest.raises(B.LambLibraryMissing):
        B.load(str(tmp_path / "missing.so"))
