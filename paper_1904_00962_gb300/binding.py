"""ctypes binding of liblamb.so -- argument marshalling only.

Every function has the name of the C entry point it wraps (include/lamb.h)
and raises LambError when the C call returns a non-zero status.  Pointers
are Python ints (device addresses, e.g. ``tensor.data_ptr()``); streams are
raw cudaStream_t handles as ints (``torch.cuda.current_stream().cuda_stream``)
or 0 for the legacy default stream.  No arithmetic of the method happens
here: every step runs in the CUDA kernels of the library.
"""
from __future__ import annotations

import ctypes
import math
import os
from ctypes import (POINTER, Structure, byref, c_char_p, c_double, c_int32,
                    c_int64, c_uint8, c_uint32, c_void_p)

import numpy as np

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_build",
                        "liblamb.so")

# status codes
LAMB_OK = 0
LAMB_ERR_INVALID_ARG = 1
LAMB_ERR_UNSUPPORTED_DTYPE = 2
LAMB_ERR_CUDA = 3
LAMB_ERR_OOM = 4
LAMB_ERR_NOT_BOUND = 5
# dtypes
LAMB_DTYPE_NONE = -1
LAMB_F32 = 0
LAMB_BF16 = 1
# phi
LAMB_PHI_IDENTITY = 0
LAMB_PHI_CLIP = 1
# flags / status bits
LAMB_FLAG_BIAS_CORRECTION = 0x1
LAMB_FLAG_INCREMENT_STEP = 0x2
LAMB_FLAG_LR_SCHEDULE = 0x4
LAMB_FLAG_GRAD_NORM = 0x8
LAMB_FLAG_SKIP_NONFINITE = 0x10
LAMB_FLAG_DECOUPLED_DECAY = 0x20
LAMB_STATUS_NONFINITE = 0x1
LAMB_STATUS_BAD_STEP = 0x2
LAMB_STATUS_GRAD_NONFINITE = 0x8
LAMB_STATUS_SKIPPED = 0x10

EXPORTED = ["lamb_plan_create", "lamb_plan_bind", "lamb_step", "lars_step",
            "lamb_plan_trust_ratios", "lamb_plan_copy_trust_ratios",
            "lamb_plan_query", "lamb_plan_get_info",
            "lamb_plan_set_timing", "lamb_plan_read_timing",
            "lamb_plan_destroy", "lamb_layout_chunks", "lamb_last_error",
            "lamb_abi_version", "lamb_step_noalloc",
            "nlamb_step", "lamb_plan_grad_norms", "lamb_plan_copy_grad_norms",
            "lamb_layout_rounds", "lamb_shard_pass1", "lamb_shard_pass2",
            "lamb_plan_partials", "lamb_layout_shard",
            "lamb_plan_copy_partials"]


class LambError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"liblamb status {status}: {message}")
        self.status = status


class LambLibraryMissing(ImportError):
    pass


class lamb_hyper_t(Structure):
    _fields_ = [("beta1", c_double), ("beta2", c_double), ("eps", c_double),
                ("weight_decay", c_double), ("gamma_l", c_double),
                ("gamma_u", c_double), ("trust_coef", c_double),
                ("phi", c_int32), ("flags", c_uint32),
                ("lr_base", c_double), ("lr_warmup_steps", c_int64),
                ("lr_total_steps", c_int64)]


LAMB_ALGO_AUTO = 0
LAMB_ALGO_TWO_PASS = 1
LAMB_ALGO_ON_CHIP = 3
LAMB_ONCHIP_ROW_ELEMS = 128       # row of an on-chip step
LAMB_TAIL_CHUNK_ELEMS = 2048      # chunks near the ends of a two-pass layout
LAMB_OPT_LAMB = 0
LAMB_OPT_LARS = 1
LAMB_OPT_NLAMB = 2
LAMB_OPT_NNLAMB = 3
LAMB_STATUS_WAIT_TIMEOUT = 0x4


class lamb_plan_options_t(Structure):
    _fields_ = [("chunk_elems", c_int32), ("blocks_per_sm", c_int32),
                ("algorithm", c_int32), ("wait_limit_ms", c_int32),
                ("test_unmet_wait", c_int32), ("onchip_max_ctas", c_int32),
                ("onchip_rows", c_int32), ("tail_elems", c_int64),
                ("shard_world", c_int32), ("shard_rank", c_int32)]


class lamb_plan_info_t(Structure):
    _fields_ = [("n_tensors", c_int32), ("n_chunks", c_int32),
                ("n_params", c_int64), ("chunk_elems", c_int32),
                ("grid_blocks", c_int32), ("threads_per_block", c_int32),
                ("num_sms", c_int32), ("device", c_int32),
                ("grad_dtype", c_int32), ("copy_dtype", c_int32),
                ("bound", c_int32), ("n_vector_tensors", c_int32),
                ("device_bytes", c_int64), ("algorithm", c_int32),
                ("n_rounds", c_int32), ("n_streamed_tensors", c_int32),
                ("rows_per_cta", c_int32), ("row_elems", c_int32),
                ("tail_elems", c_int64), ("shard_world", c_int32),
                ("shard_rank", c_int32), ("shard_chunk_begin", c_int64),
                ("shard_chunk_end", c_int64)]


_lib = None


def load(path: str | None = None) -> ctypes.CDLL:
    """Load liblamb.so once; raises LambLibraryMissing if it is not built."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise LambLibraryMissing(
            f"{p} not found: build it with `python -m "
            f"paper_1904_00962_gb300.build` (needs nvcc)")
    lib = ctypes.CDLL(p)
    vp = c_void_p
    lib.lamb_plan_create.argtypes = [POINTER(c_int64), c_int32,
                                     POINTER(c_uint8), c_int32, c_int32,
                                     c_int32, POINTER(lamb_plan_options_t),
                                     POINTER(vp)]
    lib.lamb_plan_bind.argtypes = [vp, POINTER(vp), POINTER(vp), POINTER(vp),
                                   POINTER(vp), POINTER(vp), vp]
    for name in ("lamb_step", "lars_step"):
        getattr(lib, name).argtypes = [vp, POINTER(lamb_hyper_t), vp, vp, vp]
    lib.nlamb_step.argtypes = [vp, POINTER(lamb_hyper_t), c_double, c_int32,
                               vp, vp, vp, vp]
    lib.lamb_plan_trust_ratios.argtypes = [vp, POINTER(vp), POINTER(vp),
                                           POINTER(vp)]
    lib.lamb_plan_copy_trust_ratios.argtypes = [vp, vp, vp, vp, vp]
    lib.lamb_plan_grad_norms.argtypes = [vp, POINTER(vp), POINTER(vp),
                                         POINTER(vp)]
    lib.lamb_plan_copy_grad_norms.argtypes = [vp, vp, vp, vp, vp]
    lib.lamb_plan_query.argtypes = [vp, POINTER(c_uint32), c_int32, vp]
    lib.lamb_plan_get_info.argtypes = [vp, POINTER(lamb_plan_info_t)]
    lib.lamb_plan_set_timing.argtypes = [vp, c_int32]
    lib.lamb_plan_read_timing.argtypes = [vp, POINTER(c_int32),
                                          POINTER(c_double), c_int32]
    lib.lamb_plan_destroy.argtypes = [vp]
    lib.lamb_layout_chunks.argtypes = [POINTER(c_int64), c_int32, c_int32,
                                       c_int64,
                                       POINTER(c_int32), POINTER(c_int64),
                                       POINTER(c_int32), c_int32,
                                       POINTER(c_int32)]
    lib.lamb_step_noalloc.argtypes = [POINTER(c_int64), c_int32,
                                      POINTER(c_uint8), c_int32, c_int32,
                                      POINTER(vp), POINTER(vp), POINTER(vp),
                                      POINTER(vp), POINTER(vp),
                                      POINTER(lamb_hyper_t), vp, vp, vp, vp]
    for name in ("lamb_shard_pass1", "lamb_shard_pass2"):
        getattr(lib, name).argtypes = [vp, POINTER(lamb_hyper_t), c_int32,
                                       c_double, vp, vp, vp, vp]
    lib.lamb_plan_partials.argtypes = [vp, POINTER(vp), POINTER(c_int64)]
    lib.lamb_plan_copy_partials.argtypes = [vp, vp, c_int32, vp]
    lib.lamb_layout_shard.argtypes = [POINTER(c_int64), c_int32, c_int32,
                                      c_int64, c_int32, c_int32,
                                      POINTER(c_int64), POINTER(c_int64)]
    lib.lamb_layout_rounds.argtypes = [POINTER(c_int64), c_int32, c_int32,
                                       c_int32, *([vp] * 7), c_int64,
                                       POINTER(c_int64), POINTER(c_int32)]
    for name in EXPORTED:
        if name in ("lamb_last_error", "lamb_abi_version"):
            continue
        getattr(lib, name).restype = c_int32
    lib.lamb_last_error.restype = c_char_p
    lib.lamb_last_error.argtypes = []
    lib.lamb_abi_version.restype = c_int32
    lib.lamb_abi_version.argtypes = []
    if path is None:
        _lib = lib
    return lib


def _check(status: int) -> None:
    if status != LAMB_OK:
        raise LambError(status, lamb_last_error())


def _ptr_array(ptrs):
    if ptrs is None:
        return None
    return (c_void_p * len(ptrs))(*[int(p) if p else None for p in ptrs])


def lamb_last_error() -> str:
    return load().lamb_last_error().decode()


def lamb_abi_version() -> int:
    return int(load().lamb_abi_version())


def make_hyper(*, beta1=0.9, beta2=0.999, eps=1e-6, weight_decay=0.01,
               phi="identity", gamma_l=0.0, gamma_u=math.inf, trust_coef=1.0,
               bias_correction=True, increment_step=False, lr_schedule=None,
               grad_norm=False, skip_nonfinite=False, decoupled_decay=False
               ) -> lamb_hyper_t:
    """Fill a lamb_hyper_t (plain field copy).  lr_schedule: None or
    (eta_0, warmup_steps, total_steps) for LAMB_FLAG_LR_SCHEDULE."""
    flags = (LAMB_FLAG_BIAS_CORRECTION if bias_correction else 0) | \
            (LAMB_FLAG_INCREMENT_STEP if increment_step else 0) | \
            (LAMB_FLAG_LR_SCHEDULE if lr_schedule is not None else 0) | \
            (LAMB_FLAG_GRAD_NORM if grad_norm else 0) | \
            (LAMB_FLAG_SKIP_NONFINITE if skip_nonfinite else 0) | \
            (LAMB_FLAG_DECOUPLED_DECAY if decoupled_decay else 0)
    base, warm, total = lr_schedule if lr_schedule is not None else (0.0, 0, 1)
    return lamb_hyper_t(beta1, beta2, eps, weight_decay, gamma_l, gamma_u,
                        trust_coef, LAMB_PHI_CLIP if phi == "clip"
                        else LAMB_PHI_IDENTITY, flags, float(base), int(warm),
                        int(total))


def lamb_plan_create(sizes, decay_mask=None, grad_dtype=LAMB_F32,
                     copy_dtype=LAMB_DTYPE_NONE, device=0, chunk_elems=0,
                     blocks_per_sm=0, algorithm=LAMB_ALGO_AUTO,
                     wait_limit_ms=0,
                     test_unmet_wait=False, onchip_max_ctas=0,
                     onchip_rows=0, tail_elems=0, shard_world=0,
                     shard_rank=0) -> int:
    lib = load()
    n = len(sizes)
    sz = (c_int64 * max(n, 1))(*[int(s) for s in sizes])
    mask = None
    if decay_mask is not None:
        mask = (c_uint8 * max(n, 1))(*[1 if d else 0 for d in decay_mask])
    opts = lamb_plan_options_t(int(chunk_elems), int(blocks_per_sm),
                               int(algorithm), int(wait_limit_ms),
                               int(bool(test_unmet_wait)),
                               int(onchip_max_ctas), int(onchip_rows),
                               int(tail_elems), int(shard_world),
                               int(shard_rank))
    out = c_void_p()
    _check(lib.lamb_plan_create(sz, n, mask, int(grad_dtype), int(copy_dtype),
                                int(device), byref(opts), byref(out)))
    return out.value


def lamb_plan_bind(plan, w, g, m, v=None, w_copy=None, stream=0) -> None:
    _check(load().lamb_plan_bind(c_void_p(plan), _ptr_array(w), _ptr_array(g),
                                 _ptr_array(m), _ptr_array(v),
                                 _ptr_array(w_copy), c_void_p(stream or None)))


def lamb_step(plan, hyper: lamb_hyper_t, d_step, d_lr, stream=0) -> None:
    _check(load().lamb_step(c_void_p(plan), byref(hyper),
                            c_void_p(d_step or None), c_void_p(d_lr or None),
                            c_void_p(stream or None)))


def lars_step(plan, hyper: lamb_hyper_t, d_step, d_lr, stream=0) -> None:
    _check(load().lars_step(c_void_p(plan), byref(hyper),
                            c_void_p(d_step or None), c_void_p(d_lr or None),
                            c_void_p(stream or None)))


def nlamb_step(plan, hyper: lamb_hyper_t, momentum_decay, nesterov_second_moment,
               d_step, d_lr, d_mu_product, stream=0) -> None:
    _check(load().nlamb_step(c_void_p(plan), byref(hyper),
                             float(momentum_decay),
                             int(bool(nesterov_second_moment)),
                             c_void_p(d_step or None), c_void_p(d_lr or None),
                             c_void_p(d_mu_product or None),
                             c_void_p(stream or None)))


def step_call(kind, plan, hyper: lamb_hyper_t, d_step, d_lr, stream=0,
              momentum_decay=0.0, d_mu_product=0):
    """A zero-argument callable that runs one lamb_step ("lamb"), lars_step
    ("lars") or nlamb_step ("nlamb", "nnlamb") with its arguments marshalled
    once, for loops that repeat the same step.  The callable keeps `hyper`
    alive and reads it at each call."""
    lib = load()
    p, hp = c_void_p(plan), byref(hyper)
    ds, dl = c_void_p(d_step or None), c_void_p(d_lr or None)
    s = c_void_p(stream or None)
    if kind == "lamb":
        fn, args = lib.lamb_step, (p, hp, ds, dl, s)
    elif kind == "lars":
        fn, args = lib.lars_step, (p, hp, ds, dl, s)
    elif kind in ("nlamb", "nnlamb"):
        fn, args = lib.nlamb_step, (p, hp, c_double(momentum_decay),
                                    c_int32(kind == "nnlamb"), ds, dl,
                                    c_void_p(d_mu_product or None), s)
    else:
        raise ValueError(f"unknown step kind {kind!r}")

    def call():
        st = fn(*args)
        if st:
            _check(st)
    return call


def lamb_plan_trust_ratios(plan):
    r, w, u = c_void_p(), c_void_p(), c_void_p()
    _check(load().lamb_plan_trust_ratios(c_void_p(plan), byref(r), byref(w),
                                         byref(u)))
    return r.value, w.value, u.value


def lamb_plan_grad_norms(plan):
    """Device addresses of (||g_k|| [n] f64, global ||g|| [1] f64,
    non-finite flag [1] u32)."""
    a, b, c = c_void_p(), c_void_p(), c_void_p()
    _check(load().lamb_plan_grad_norms(c_void_p(plan), byref(a), byref(b),
                                       byref(c)))
    return a.value, b.value, c.value


def lamb_plan_copy_grad_norms(plan, gnorm=0, gnorm_global=0, nonfinite=0,
                              stream=0) -> None:
    """Addresses (device or host) of caller-owned arrays, or 0."""
    _check(load().lamb_plan_copy_grad_norms(
        c_void_p(plan), c_void_p(gnorm or None), c_void_p(gnorm_global or None),
        c_void_p(nonfinite or None), c_void_p(stream or None)))


def lamb_plan_copy_trust_ratios(plan, ratio=0, wnorm=0, unorm=0,
                                stream=0) -> None:
    """Addresses (device or host) of caller-owned float64 arrays, or 0."""
    _check(load().lamb_plan_copy_trust_ratios(
        c_void_p(plan), c_void_p(ratio or None), c_void_p(wnorm or None),
        c_void_p(unorm or None), c_void_p(stream or None)))


def lamb_plan_query(plan, clear=False, stream=0) -> int:
    bits = c_uint32()
    _check(load().lamb_plan_query(c_void_p(plan), byref(bits), int(clear),
                                  c_void_p(stream or None)))
    return int(bits.value)


def lamb_plan_get_info(plan) -> dict:
    info = lamb_plan_info_t()
    _check(load().lamb_plan_get_info(c_void_p(plan), byref(info)))
    return {name: getattr(info, name) for name, _ in info._fields_}


def lamb_plan_set_timing(plan, enable=True) -> None:
    _check(load().lamb_plan_set_timing(c_void_p(plan), int(bool(enable))))


def lamb_plan_read_timing(plan, n_kernels=2):
    n = c_int32()
    ms = (c_double * n_kernels)()
    _check(load().lamb_plan_read_timing(c_void_p(plan), byref(n), ms,
                                        n_kernels))
    return int(n.value), [float(x) for x in ms]


def lamb_plan_destroy(plan) -> None:
    if plan:
        _check(load().lamb_plan_destroy(c_void_p(plan)))


def lamb_step_noalloc(sizes, decay_mask, grad_dtype, copy_dtype, w, g, m, v,
                      w_copy, hyper: lamb_hyper_t, d_step, d_lr, d_ratio=0,
                      stream=0) -> None:
    """Allocation-free LAMB step (see include/lamb.h): pointer lists as in
    lamb_plan_bind, d_ratio an optional device float64 array."""
    n = len(sizes)
    sz = (c_int64 * max(n, 1))(*[int(s) for s in sizes])
    mask = None
    if decay_mask is not None:
        mask = (c_uint8 * max(n, 1))(*[1 if d else 0 for d in decay_mask])
    _check(load().lamb_step_noalloc(
        sz, n, mask, int(grad_dtype), int(copy_dtype), _ptr_array(w),
        _ptr_array(g), _ptr_array(m), _ptr_array(v), _ptr_array(w_copy),
        byref(hyper), c_void_p(d_step or None), c_void_p(d_lr or None),
        c_void_p(d_ratio or None), c_void_p(stream or None)))


def lamb_layout_chunks(sizes, chunk_elems=0, tail_elems=0):
    """Host-only planner: returns (tensor, offset, length) int arrays."""
    lib = load()
    n = len(sizes)
    sz = (c_int64 * max(n, 1))(*[int(s) for s in sizes])
    count = c_int32()
    st = lib.lamb_layout_chunks(sz, n, int(chunk_elems), int(tail_elems),
                                None, None, None, 0,
                                byref(count))
    _check(st)
    cap = count.value
    t = np.zeros(max(cap, 1), dtype=np.int32)
    o = np.zeros(max(cap, 1), dtype=np.int64)
    ln = np.zeros(max(cap, 1), dtype=np.int32)
    _check(lib.lamb_layout_chunks(
        sz, n, int(chunk_elems), int(tail_elems),
        t.ctypes.data_as(POINTER(c_int32)),
        o.ctypes.data_as(POINTER(c_int64)), ln.ctypes.data_as(POINTER(c_int32)),
        cap, byref(count)))
    return t[:cap], o[:cap], ln[:cap]


def lamb_layout_rounds(sizes, grid, rows_per_cta):
    """Host-only: the pieces of an on-chip plan as a dict of arrays (round,
    cta, tensor, offset, len, first_row, rows) and the round count."""
    lib = load()
    n = len(sizes)
    sz = (c_int64 * max(n, 1))(*[int(s) for s in sizes])
    count, rounds = c_int64(), c_int32()
    _check(lib.lamb_layout_rounds(sz, n, int(grid), int(rows_per_cta),
                                  *([None] * 7), 0, byref(count),
                                  byref(rounds)))
    cap = count.value
    out = {"round": np.zeros(max(cap, 1), np.int32),
           "cta": np.zeros(max(cap, 1), np.int32),
           "tensor": np.zeros(max(cap, 1), np.int32),
           "offset": np.zeros(max(cap, 1), np.int64),
           "len": np.zeros(max(cap, 1), np.int64),
           "first_row": np.zeros(max(cap, 1), np.int32),
           "rows": np.zeros(max(cap, 1), np.int32)}
    _check(lib.lamb_layout_rounds(
        sz, n, int(grid), int(rows_per_cta),
        *[out[k].ctypes.data for k in ("round", "cta", "tensor", "offset",
                                        "len", "first_row", "rows")],
        cap, byref(count), byref(rounds)))
    return {k: v[:cap] for k, v in out.items()}, int(rounds.value)


def lamb_shard_pass1(plan, hyper: lamb_hyper_t, optimizer=LAMB_OPT_LAMB,
                     momentum_decay=0.0, d_step=0, d_lr=0, d_mu_product=0,
                     stream=0) -> None:
    _check(load().lamb_shard_pass1(c_void_p(plan), byref(hyper),
                                   int(optimizer), float(momentum_decay),
                                   c_void_p(d_step or None),
                                   c_void_p(d_lr or None),
                                   c_void_p(d_mu_product or None),
                                   c_void_p(stream or None)))


def lamb_shard_pass2(plan, hyper: lamb_hyper_t, optimizer=LAMB_OPT_LAMB,
                     momentum_decay=0.0, d_step=0, d_lr=0, d_mu_product=0,
                     stream=0) -> None:
    _check(load().lamb_shard_pass2(c_void_p(plan), byref(hyper),
                                   int(optimizer), float(momentum_decay),
                                   c_void_p(d_step or None),
                                   c_void_p(d_lr or None),
                                   c_void_p(d_mu_product or None),
                                   c_void_p(stream or None)))


def lamb_plan_partials(plan):
    """(device address of the float sums array, number of floats)."""
    ptr, n = c_void_p(), c_int64()
    _check(load().lamb_plan_partials(c_void_p(plan), byref(ptr), byref(n)))
    return ptr.value, int(n.value)


def lamb_layout_shard(sizes, world, rank, chunk_elems=0, tail_elems=0):
    """Host-only: chunk range (begin, end) of shard `rank` of `world`."""
    n = len(sizes)
    sz = (c_int64 * max(n, 1))(*[int(s) for s in sizes])
    b, e = c_int64(), c_int64()
    _check(load().lamb_layout_shard(sz, n, int(chunk_elems), int(tail_elems),
                                    int(world), int(rank), byref(b),
                                    byref(e)))
    return int(b.value), int(e.value)


def lamb_plan_copy_partials(plan, buf, to_plan, stream=0) -> None:
    """Copy the plan's sums array to (to_plan false) or from (true) the
    device or host address buf."""
    _check(load().lamb_plan_copy_partials(c_void_p(plan), c_void_p(buf),
                                          int(bool(to_plan)),
                                          c_void_p(stream or None)))
