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


def test_binding_constants_match_header_defines():
    # every #define LAMB_* value the binding mirrors must agree with the ABI
    hdr = open(os.path.join(ROOT, "include", "lamb.h")).read()
    defs = dict(re.findall(r"#define\s+(LAMB_[A-Z0-9_]+)\s+(0x[0-9a-fA-F]+|\d+)u?\b",
                           hdr))
    checked = 0
    for name, val in defs.items():
        if hasattr(B, name):
            assert getattr(B, name) == int(val, 0), name
            checked += 1
    assert checked >= 12
    for flag in ("LAMB_FLAG_GRAD_NORM", "LAMB_FLAG_SKIP_NONFINITE",
                 "LAMB_FLAG_DECOUPLED_DECAY", "LAMB_ONCHIP_ROW_ELEMS",
                 "LAMB_STATUS_SKIPPED"):
        assert flag in defs and hasattr(B, flag), flag
    # and every enumerator (status codes, dtypes, phi) by name and value
    enums = dict(re.findall(r"\b(LAMB_[A-Z0-9_]+)\s*=\s*(-?\d+)", hdr))
    assert len(enums) == 11
    for name, val in enums.items():
        assert getattr(B, name) == int(val), name


def test_binding_signatures_match_the_header(lib):
    """Every declared entry point's ctypes argtypes have the declaration's
    arity, the same integer width or double for each scalar, and a pointer
    for each pointer (plans and streams are pointers too)."""
    text = open(HEADER).read()
    decls = re.findall(r"LAMB_API\s+[\w\s\*]+?\b(\w+)\s*\(([^)]*)\)\s*;",
                       text, re.S)
    assert len(decls) == len(_declared())
    scalar = {"int32_t": ctypes.c_int32, "int64_t": ctypes.c_int64,
              "double": ctypes.c_double}
    for name, params in decls:
        ps = [p.strip() for p in params.split(",")]
        ps = [] if ps == ["void"] else ps
        at = getattr(lib, name).argtypes or []
        assert len(at) == len(ps), name
        for p, t in zip(ps, at):
            base = p.replace("const", "").split()[0]
            if "*" in p or base in ("lamb_plan_t", "cudaStream_t"):
                assert t in (ctypes.c_void_p, ctypes.c_char_p) or \
                    issubclass(t, ctypes._Pointer), (name, p)
            else:
                assert t is scalar[base], (name, p)


def test_abi_version(lib):
    assert B.lamb_abi_version() == 3


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


def test_c_program_links_and_plans(lib, tmp_path):
    """A plain C99 program, linked against the shared library with nothing
    but include/lamb.h, uses the host-only entry points: the ABI version,
    the chunk table, a shard range and the on-chip rounds of a small layout,
    and a rejected plan creation with its error message."""
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("gcc not available")
    src = tmp_path / "user.c"
    src.write_text(r"""
#include <stdio.h>
#include <string.h>
#include "lamb.h"
int main(void) {
  const int64_t sizes[4] = {1000000, 1024, 0, 70000};
  int32_t t[128], len[128], n = 0;
  int64_t off[128], total = 0, b = 0, e = 0;
  if (lamb_abi_version() != LAMB_ABI_VERSION) return 10;
  if (lamb_layout_chunks(sizes, 4, 16384, 0, t, off, len, 128, &n) != LAMB_OK)
    return 11;
  for (int i = 0; i < n; ++i) total += len[i];
  if (total != 1071024) return 12;
  if (lamb_layout_shard(sizes, 4, 16384, 0, 2, 1, &b, &e) != LAMB_OK)
    return 13;
  int64_t pieces = 0;
  int32_t rounds = 0;
  if (lamb_layout_rounds(sizes, 4, 152, 216, NULL, NULL, NULL, NULL, NULL,
                         NULL, NULL, 0, &pieces, &rounds) != LAMB_OK)
    return 14;                     /* capacity 0: the counts only */
  lamb_plan_t plan = NULL;
  if (lamb_plan_create(NULL, 4, NULL, LAMB_F32, LAMB_DTYPE_NONE, 0, NULL,
                       &plan) !=
      LAMB_ERR_INVALID_ARG || plan != NULL || strlen(lamb_last_error()) == 0)
    return 15;
  printf("%d %lld %lld %lld %d\n", n, (long long)b, (long long)e,
         (long long)pieces, rounds);
  return 0;
}
""")
    build_dir = os.path.dirname(B.LIB_PATH)
    exe = tmp_path / "user"
    res = subprocess.run([gcc, "-std=c99", "-Wall", "-Werror",
                          "-I", os.path.join(ROOT, "include"),
                          "-I", "/usr/local/cuda/include", str(src),
                          "-o", str(exe), "-L", build_dir, "-llamb",
                          "-Wl,-rpath," + build_dir],
                         capture_output=True, text=True)
    assert res.returncode == 0, res.stderr
    run = subprocess.run([str(exe)], capture_output=True, text=True,
                         timeout=60)
    assert run.returncode == 0, (run.returncode, run.stderr)
    n, b, e, pieces, rounds = map(int, run.stdout.split())
    t, o, ln = B.lamb_layout_chunks([1000000, 1024, 0, 70000], 16384)
    assert n == len(t)
    assert (b, e) == B.lamb_layout_shard([1000000, 1024, 0, 70000], 2, 1,
                                         16384, 0)
    p, n_rounds = B.lamb_layout_rounds([1000000, 1024, 0, 70000], 152, 216)
    assert (pieces, rounds) == (len(p["round"]), n_rounds)


def test_struct_layouts_match_ctypes(tmp_path):
    """sizeof and field offsets of the ABI structs, as a C compiler lays
    them out from include/lamb.h, equal the ctypes mirrors in binding.py."""
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("gcc not available")
    structs = [("lamb_hyper_t", B.lamb_hyper_t),
               ("lamb_plan_options_t", B.lamb_plan_options_t),
               ("lamb_plan_info_t", B.lamb_plan_info_t)]
    lines = ['#include <stdio.h>', '#include <stddef.h>', '#include "lamb.h"',
             'int main(void){']
    for cname, ct in structs:
        lines.append(f'printf("{cname} %zu\\n", sizeof({cname}));')
        for f, _ in ct._fields_:
            lines.append(f'printf("{cname}.{f} %zu\\n", offsetof({cname}, {f}));')
    lines.append("return 0;}")
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines))
    exe = tmp_path / "layout"
    res = subprocess.run([gcc, "-std=c99", "-I", os.path.join(ROOT, "include"),
                          "-I", "/usr/local/cuda/include", str(src), "-o",
                          str(exe)], capture_output=True, text=True)
    assert res.returncode == 0, res.stderr
    out = dict(l.split() for l in subprocess.run(
        [str(exe)], capture_output=True, text=True).stdout.splitlines())
    for cname, ct in structs:
        assert int(out[cname]) == ctypes.sizeof(ct), cname
        for f, _ in ct._fields_:
            assert int(out[f"{cname}.{f}"]) == getattr(ct, f).offset, (cname, f)


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
    st = lib.lamb_layout_chunks(sz, 1, 1024, 0, t, o, ln, 2, ctypes.byref(n))
    assert st == B.LAMB_ERR_INVALID_ARG and n.value == 10


@pytest.mark.parametrize("tail", [1, 2048, 5000, 100000, 10 ** 9])
def test_chunk_table_tail_chunks(lib, tail):
    """Within `tail` elements of either end of the layout (tensors laid end
    to end) the chunks are short; elsewhere they are full; every element is
    covered once, in tensor order, and no chunk spans two tensors."""
    rng = np.random.default_rng(tail)
    sizes = [0, 3, 70000, 1, 16384 * 5 + 7, *rng.integers(1, 90000, 20).tolist(),
             33000, 0]
    chunk, small = 16384, B.LAMB_TAIL_CHUNK_ELEMS
    t, o, ln = B.lamb_layout_chunks(sizes, chunk, tail)
    total = sum(sizes)
    starts = np.concatenate([[0], np.cumsum(sizes)[:-1]])
    pos = starts[t] + o                          # position in the layout
    assert np.all(np.diff(t) >= 0) and np.all(o % 1024 == 0)
    for k, s in enumerate(sizes):
        sel = t == k
        if s == 0:
            assert not sel.any()
            continue
        offs, lens = o[sel], ln[sel]
        assert offs[0] == 0 and offs[-1] + lens[-1] == s
        np.testing.assert_array_equal(offs[1:], offs[:-1] + lens[:-1])
    in_tail = (pos < tail) | (pos + chunk > total - tail)
    assert np.all(ln[in_tail] <= small)
    # away from the ends a chunk is short only where its tensor ends
    ends = pos + ln == starts[t] + np.asarray(sizes)[t]
    assert np.all((ln[~in_tail] == chunk) | ends[~in_tail])
    if tail >= total:
        assert np.all(ln <= small)


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
    with pytest.raises(B.LambError) as ei:   # a tail needs 2048+ chunks
        B.lamb_plan_create([10], chunk_elems=1024, tail_elems=5000)
    assert ei.value.status == B.LAMB_ERR_INVALID_ARG
    for bad in (dict(tail_elems=-1), dict(wait_limit_ms=-1),
                dict(algorithm=2), dict(blocks_per_sm=-1),
                dict(onchip_rows=-1), dict(shard_world=2, shard_rank=2),
                dict(shard_world=0, shard_rank=1)):
        with pytest.raises(B.LambError) as ei:
            B.lamb_plan_create([10], **bad)
        assert ei.value.status == B.LAMB_ERR_INVALID_ARG, bad



def test_noalloc_validates_before_touching_the_device(lib):
    """Every rejection of the allocation-free step happens on the host, before
    any CUDA call: the pointers below are never dereferenced (no case here is
    valid, so none reaches the device)."""
    P = 1 << 20                                   # fake, 16-byte aligned
    hyp = B.make_hyper()                          # bias correction on

    def call(sizes=(8, 8), grad=B.LAMB_F32, copy=B.LAMB_DTYPE_NONE, ptr=P,
             w_copy=None, hyper=hyp, d_step=P, d_lr=P):
        n = len(sizes)
        B.lamb_step_noalloc(list(sizes), None, grad, copy, [ptr] * n,
                            [ptr] * n, [ptr] * n, [ptr] * n, w_copy, hyper,
                            d_step, d_lr)

    cases = [
        (dict(sizes=()), B.LAMB_ERR_INVALID_ARG, "n_tensors"),
        (dict(sizes=(1,) * 4097), B.LAMB_ERR_INVALID_ARG, "4096"),
        (dict(sizes=(8, -1)), B.LAMB_ERR_INVALID_ARG, "negative"),
        (dict(sizes=((1 << 31) + 1,)), B.LAMB_ERR_INVALID_ARG, "exceeds"),
        # sizes near INT64_MAX must not wrap around the chunk count
        (dict(sizes=((1 << 63) - 1,)), B.LAMB_ERR_INVALID_ARG, "exceeds"),
        (dict(sizes=((1 << 63) - 16384,)), B.LAMB_ERR_INVALID_ARG, "exceeds"),
        (dict(sizes=(1 << 30, 1 << 30, 1)), B.LAMB_ERR_INVALID_ARG, "chunks"),
        (dict(grad=7), B.LAMB_ERR_UNSUPPORTED_DTYPE, "grad_dtype"),
        (dict(copy=B.LAMB_F32), B.LAMB_ERR_UNSUPPORTED_DTYPE, "copy_dtype"),
        (dict(copy=B.LAMB_BF16), B.LAMB_ERR_INVALID_ARG, "w_copy"),
        (dict(hyper=B.make_hyper(beta1=1.0)), B.LAMB_ERR_INVALID_ARG, "hyper"),
        (dict(hyper=B.make_hyper(grad_norm=True)), B.LAMB_ERR_INVALID_ARG,
         "hyper"),
        (dict(d_step=0), B.LAMB_ERR_INVALID_ARG, "d_step"),
        (dict(d_lr=0), B.LAMB_ERR_INVALID_ARG, "d_lr"),
        (dict(ptr=0), B.LAMB_ERR_INVALID_ARG, "NULL"),
        (dict(ptr=P + 2), B.LAMB_ERR_INVALID_ARG, "aligned"),
    ]
    for kw, status, word in cases:
        with pytest.raises(B.LambError) as ei:
            call(**kw)
        assert ei.value.status == status, kw
        assert word in B.lamb_last_error(), (kw, B.lamb_last_error())

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


# ---------------------------------------------------------------------------
# On-chip round planner (host only)
# ---------------------------------------------------------------------------

def _check_rounds(sizes, grid, rpc):
    p, n_rounds = B.lamb_layout_rounds(sizes, grid, rpc)
    row = B.LAMB_ONCHIP_ROW_ELEMS
    # a resident tensor has at most 65,535 rows (the kernel's row records)
    cap = min(grid * rpc, 65535)
    rows_of = [(s + row - 1) // row for s in sizes]
    streamed = p["round"] < 0
    # tensors too large for a round are streamed whole, and only those
    np.testing.assert_array_equal(
        np.sort(p["tensor"][streamed]),
        [k for k, r in enumerate(rows_of) if r > cap])
    assert np.all(p["len"][streamed] == np.asarray(sizes)[p["tensor"][streamed]])
    on = ~streamed
    # every element of every other non-empty tensor is in exactly one piece,
    # in order, whole rows except at the tensor's end, all in one round
    for k, s in enumerate(sizes):
        if rows_of[k] == 0 or rows_of[k] > cap:
            assert not np.any(p["tensor"][on] == k), k
            continue
        sel = np.flatnonzero(on & (p["tensor"] == k))
        off, ln = p["offset"][sel], p["len"][sel]
        assert off[0] == 0 and off[-1] + ln[-1] == s, k
        np.testing.assert_array_equal(off[1:], off[:-1] + ln[:-1])
        assert np.all(off % row == 0)
        assert np.all(p["rows"][sel] == (ln + row - 1) // row)
        assert len(set(p["round"][sel].tolist())) == 1, k
    # per (round, CTA): at most 16 pieces, rows packed from 0, within rpc
    assert 0 <= p["round"][on].min(initial=0) and \
        p["round"][on].max(initial=-1) < n_rounds
    assert np.all((p["cta"][on] >= 0) & (p["cta"][on] < grid))
    for r in range(n_rounds):
        for c in np.unique(p["cta"][on & (p["round"] == r)]):
            sel = np.flatnonzero(on & (p["round"] == r) & (p["cta"] == c))
            assert len(sel) <= 16
            fr, nr = p["first_row"][sel], p["rows"][sel]
            assert fr[0] == 0
            np.testing.assert_array_equal(fr[1:], fr[:-1] + nr[:-1])
            assert fr[-1] + nr[-1] <= rpc
    return p, n_rounds


@pytest.mark.parametrize("grid,rpc", [(152, 216), (152, 217), (4, 8),
                                      (7, 3), (1, 224)])
def test_rounds_cover_every_tensor_once(lib, grid, rpc):
    rng = np.random.default_rng(grid * 1000 + rpc)
    sizes = [0, 1, 127, 128, 129, 4096, 100003] + \
        rng.integers(0, 3 * 128 * rpc, 60).tolist()
    _check_rounds(sizes, grid, rpc)


def test_rounds_stream_tensors_beyond_65535_rows(lib):
    row = B.LAMB_ONCHIP_ROW_ELEMS
    sizes = [65535 * row, 65536 * row - 5, 10, 70000 * row]
    p, n = _check_rounds(sizes, 400, 224)      # 89,600 rows per round
    assert sorted(p["tensor"][p["round"] < 0].tolist()) == [1, 3]


def test_rounds_of_the_paper_layouts(lib):
    from paper_1904_00962_gb300.workloads import (bert_large_layout,
                                                   resnet50_layout)
    p, n = _check_rounds(resnet50_layout().sizes, 152, 216)
    assert n == 7 and not np.any(p["round"] < 0)
    p, n = _check_rounds(bert_large_layout().sizes, 152, 216)
    # only the word embedding (30522 x 1024) is streamed
    assert n == 74 and p["tensor"][p["round"] < 0].tolist() == [0]


def test_rounds_reject_bad_input(lib):
    for args in (([10], 0, 8), ([10], 4, 0), ([10], 4, 225), ([-1], 4, 8)):
        with pytest.raises(B.LambError):
            B.lamb_layout_rounds(*args)


def test_step_call_rejects_an_unknown_step(lib):
    hyper = B.make_hyper()
    with pytest.raises(ValueError):
        B.step_call("adamw", 0, hyper, 0, 0)
