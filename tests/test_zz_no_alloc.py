"""GPU test of lamb_step_noalloc, the LAMB entry point for callers that may
not allocate device memory (e.g. code running under a framework allocator
that owns all GPU memory, or code that must avoid the device-wide
synchronisation of cudaMalloc).  Its results must match the plan-based
lamb_step on identical inputs, on two calls in a row (the second call runs
on whatever the first left in the shared device scratch).

This file is named to be collected last, so a run that stops at the first
failure has already run every other test."""
import numpy as np
import pytest
import torch

from gpu_util import TOL_RATIO, TOL_STEP, GpuLayout, c_hyper, f32
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


def _close(a, b, tol):
    a = a.double()
    b = b.double()
    scale = torch.maximum(a.abs(), b.abs())
    return bool(torch.all((a - b).abs() <= tol * scale))


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
    ref = GpuLayout(L)                       # existing entry point (plan)
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
        for name in ("w", "m", "v"):
            assert _close(getattr(st, name), getattr(ref.st, name), TOL_STEP), \
                (call, name)
        if copy_dtype:
            assert torch.equal(st.copy.view(torch.int16),
                               ref.st.copy.view(torch.int16)), call
        want = ref.plan.results()[0]
        torch.cuda.synchronize()
        assert _close(ratio, want, TOL_RATIO), call
        assert int(d_step.item()) == int(ref.d_step.item()) == 7 + call
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
    assert "chunks" in B.lamb_last_error()
    # a valid call afterwards still works
    B.lamb_step_noalloc([4], None, B.LAMB_F32, B.LAMB_DTYPE_NONE,
                        st.ptrs("w"), st.ptrs("g"), st.ptrs("m"),
                        st.ptrs("v"), None, hyp, d_step.data_ptr(),
                        d_lr.data_ptr())
    torch.cuda.synchronize()
