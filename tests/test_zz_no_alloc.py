"""GPU test of lamb_step_noalloc, the LAMB entry point for callers that may
not allocate device memory (e.g. code running under a framework allocator
that owns all GPU memory, or code that must avoid the device-wide
synchronisation of cudaMalloc).  It runs the two-pass kernels on the same
16384-element chunking as a two-pass plan, so its results must equal the
plan-based lamb_step bit for bit on identical inputs, on two calls in a row
(the second call runs on whatever the first left in the shared device
scratch), and follow the fp64 oracle within the parity tolerances.

This file is named to be collected last, so a run that stops at the first
failure has already run every other test."""
import numpy as np
import pytest
import torch

from gpu_util import (TOL_STEP, GpuLayout, c_hyper, check_copy, compare_lamb,
                      f32, hyper_kwargs, ratio_ok)
from oracle import lamb_oracle as O
from paper_1904_00962_gb300 import binding as B
from paper_1904_00962_gb300 import build as build_mod
from paper_1904_00962_gb300 import workloads as W
from paper_1904_00962_gb300.state import DeviceState

pytestmark = pytest.mark.gpu

SIZES = [0, 1, 3, 1023, 16383, 16384, 16385, 65539, 5, 100003, 2, 40000]


def _layout(grad_dtype, copy_dtype):
    n = len(SIZES)
    return W.Layout(name="noalloc", names=[f"t{i}" for i in range(n)],
                    shapes=[(s,) for s in SIZES],
                    decay=[(i + 1) % 2 for i in range(n)],
                    init=[("normal", 0.02)] * n,
                    grad_sigma=[10 ** (-2 - (i % 3)) for i in range(n)],
                    grad_dtype=grad_dtype, copy_dtype=copy_dtype,
                    zero_w={3}, zero_g={6},
                    hyper=W.Hyper(lr=2e-3, phi="clip", gamma_l=0.0,
                                  gamma_u=10.0))


def _bits(t):
    return t.view(torch.int16) if t.dtype == torch.bfloat16 else t


@pytest.fixture(scope="module")
def lib(gpu):
    build_mod.build()
    return B.load()


@pytest.mark.parametrize("grad_dtype,copy_dtype", [("f32", None),
                                                    ("bf16", "bf16")])
def test_noalloc_matches_plan_step_on_two_calls(lib, grad_dtype, copy_dtype):
    L = _layout(grad_dtype, copy_dtype)
    h = L.hyper
    hyp = c_hyper(h, increment=True)
    ref = GpuLayout(L, algorithm=B.LAMB_ALGO_TWO_PASS)   # the plan entry point
    ref.load_weights()
    ref.load_warm_state()
    st = DeviceState(L.sizes, grad_dtype=grad_dtype, copy_dtype=copy_dtype)
    for name in ("w", "m", "v"):
        getattr(st, name).copy_(getattr(ref.st, name))
    d_step = torch.full((1,), 7, dtype=torch.int64, device="cuda:0")
    d_lr = torch.full((1,), f32(h.lr), dtype=torch.float32, device="cuda:0")
    ref.d_step.fill_(7)
    ref.d_lr.fill_(f32(h.lr))
    ratio = torch.empty(L.n_tensors, dtype=torch.float64, device="cuda:0")
    gcode = B.LAMB_BF16 if grad_dtype == "bf16" else B.LAMB_F32
    ccode = B.LAMB_BF16 if copy_dtype == "bf16" else B.LAMB_DTYPE_NONE
    stream = torch.cuda.current_stream().cuda_stream
    for call in (1, 2):
        ref.load_grads(call)
        st.g.copy_(ref.st.g)
        ref.plan.lamb_step(hyp, ref.d_step, ref.d_lr)
        B.lamb_step_noalloc(L.sizes, L.decay, gcode, ccode, st.ptrs("w"),
                            st.ptrs("g"), st.ptrs("m"), st.ptrs("v"),
                            st.ptrs("copy"), hyp, d_step.data_ptr(),
                            d_lr.data_ptr(), ratio.data_ptr(), stream)
        torch.cuda.synchronize()
        names = ("w", "m", "v") + (("copy",) if copy_dtype else ())
        for name in names:
            assert torch.equal(_bits(getattr(st, name)),
                               _bits(getattr(ref.st, name))), (call, name)
        want = ref.plan.results()[0]
        torch.cuda.synchronize()
        assert torch.equal(ratio, want), call
        assert int(d_step.item()) == int(ref.d_step.item()) == 7 + call
        if call == 1:   # and the oracle on the same inputs
            for k in range(L.n_tensors):
                w, g = L.weights(k), L.grad(k, 1)
                m, v = L.state_warm(k)
                o = O.lamb_tensor(w, g, m, v, t=7, lr=f32(h.lr),
                                  decay=bool(L.decay[k]), g_dtype=grad_dtype,
                                  **hyper_kwargs(h))
                e = compare_lamb(st.download("w", k), st.download("m", k),
                                 st.download("v", k), o, w, m,
                                 O.to_f64(g, grad_dtype), h.beta1, TOL_STEP,
                                 upd=(h, 7, f32(h.lr),
                                      h.weight_decay * L.decay[k]))
                if copy_dtype:
                    check_copy(st.download("copy", k), st.download("w", k),
                               o.w, sw=e["_sw"])
                assert ratio_ok(float(ratio[k]), o.ratio), k
    ref.close()


def test_noalloc_rejects_inputs_beyond_its_limits(lib):
    L = _layout("f32", None)
    st = DeviceState([4], device="cuda:0")
    hyp = c_hyper(L.hyper)
    d_step = torch.ones(1, dtype=torch.int64, device="cuda:0")
    d_lr = torch.ones(1, dtype=torch.float32, device="cuda:0")
    p = st.ptrs("w")[0]
    with pytest.raises(B.LambError) as ei:            # too many tensors
        B.lamb_step_noalloc([4] * 4097, None, B.LAMB_F32, B.LAMB_DTYPE_NONE,
                            [p] * 4097, [p] * 4097, [p] * 4097, [p] * 4097,
                            None, hyp, d_step.data_ptr(), d_lr.data_ptr())
    assert ei.value.status == B.LAMB_ERR_INVALID_ARG
    assert "4096" in B.lamb_last_error()
    with pytest.raises(B.LambError) as ei:            # too many chunks
        B.lamb_step_noalloc([(1 << 31) + 1], None, B.LAMB_F32,
                            B.LAMB_DTYPE_NONE, [p], [p], [p], [p], None, hyp,
                            d_step.data_ptr(), d_lr.data_ptr())
    assert ei.value.status == B.LAMB_ERR_INVALID_ARG
    assert "exceeds" in B.lamb_last_error()
    # a valid call afterwards still works
    B.lamb_step_noalloc([4], None, B.LAMB_F32, B.LAMB_DTYPE_NONE,
                        st.ptrs("w"), st.ptrs("g"), st.ptrs("m"),
                        st.ptrs("v"), None, hyp, d_step.data_ptr(),
                        d_lr.data_ptr())
    torch.cuda.synchronize()
