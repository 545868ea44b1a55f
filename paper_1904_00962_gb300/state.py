"""Device-resident optimizer state for a list of tensors (PyTorch plumbing).

PyTorch only allocates device memory and supplies streams here.  Each of
w, g, m, v (and the optional bf16 weight copy) is ONE flat device buffer;
tensor k lives at an element offset rounded up to 64 elements, so every
tensor starts on a 256-byte boundary and takes the library's vectorised
path.  ``LambPlan`` couples a plan handle of the C library with such a state
and forwards steps to the C entry points; it does no arithmetic.
"""
from __future__ import annotations

import numpy as np
import torch

from . import binding as B

ALIGN_ELEMS = 64


def _dtype_code(name):
    return {None: B.LAMB_DTYPE_NONE, "f32": B.LAMB_F32,
            "bf16": B.LAMB_BF16}[name]


class DeviceState:
    def __init__(self, sizes, *, grad_dtype="f32", copy_dtype=None,
                 device="cuda:0", with_v=True, align_elems=ALIGN_ELEMS,
                 misalign=None):
        """misalign: optional set of tensor indices placed at an odd element
        offset (+1) to exercise the element-wise path."""
        self.sizes = [int(s) for s in sizes]
        self.grad_dtype = grad_dtype
        self.copy_dtype = copy_dtype
        self.device = torch.device(device)
        offs, cur = [], 0
        misalign = misalign or set()
        for k, s in enumerate(self.sizes):
            cur = (cur + align_elems - 1) // align_elems * align_elems
            if k in misalign:
                cur += 1
            offs.append(cur)
            cur += s
        self.offsets = offs
        self.total = max(cur + align_elems, 1)
        f32 = torch.float32
        dev = self.device
        self.w = torch.zeros(self.total, dtype=f32, device=dev)
        self.m = torch.zeros(self.total, dtype=f32, device=dev)
        self.v = torch.zeros(self.total, dtype=f32, device=dev) if with_v else None
        gdt = torch.bfloat16 if grad_dtype == "bf16" else f32
        self.g = torch.zeros(self.total, dtype=gdt, device=dev)
        self.copy = (torch.zeros(self.total, dtype=torch.bfloat16, device=dev)
                     if copy_dtype == "bf16" else None)

    # -- per-tensor views and pointers ---------------------------------------
    def view(self, name: str, k: int) -> torch.Tensor:
        buf = getattr(self, name)
        o = self.offsets[k]
        return buf[o:o + self.sizes[k]]

    def ptrs(self, name: str):
        buf = getattr(self, name)
        if buf is None:
            return None
        base = buf.data_ptr()
        es = buf.element_size()
        return [base + es * o for o in self.offsets]

    # -- host <-> device -----------------------------------------------------
    def upload(self, name: str, k: int, arr: np.ndarray) -> None:
        dst = self.view(name, k)
        if dst.dtype == torch.bfloat16:
            src = torch.from_numpy(np.ascontiguousarray(arr).view(np.int16))
            dst.view(torch.int16).copy_(src)
        else:
            dst.copy_(torch.from_numpy(np.ascontiguousarray(arr)))

    def download(self, name: str, k: int) -> np.ndarray:
        t = self.view(name, k)
        if t.dtype == torch.bfloat16:
            return t.view(torch.int16).cpu().numpy().view(np.uint16)
        return t.cpu().numpy()


class LambPlan:
    """A C-library plan bound to a DeviceState."""

    def __init__(self, state: DeviceState, decay_mask=None, *, device=None,
                 chunk_elems=0, blocks_per_sm=0, algorithm=0, wait_limit_ms=0,
                 test_unmet_wait=False,
                 onchip_max_ctas=0, onchip_rows=0, tail_elems=0,
                 shard_world=0, shard_rank=0):
        self.state = state
        dev = state.device.index if device is None else device
        self.handle = B.lamb_plan_create(
            state.sizes, decay_mask, _dtype_code(state.grad_dtype),
            _dtype_code(state.copy_dtype), dev or 0, chunk_elems,
            blocks_per_sm, algorithm, wait_limit_ms,
            test_unmet_wait, onchip_max_ctas, onchip_rows, tail_elems,
            shard_world, shard_rank)
        self.n = len(state.sizes)
        self.bind()

    def bind(self, stream=None):
        s = self.state
        B.lamb_plan_bind(self.handle, s.ptrs("w"), s.ptrs("g"), s.ptrs("m"),
                         s.ptrs("v"), s.ptrs("copy"), _stream(stream))

    def lamb_step(self, hyper, d_step: torch.Tensor, d_lr: torch.Tensor,
                  stream=None):
        B.lamb_step(self.handle, hyper,
                    d_step.data_ptr() if d_step is not None else 0,
                    d_lr.data_ptr(), _stream(stream))

    def lars_step(self, hyper, d_step, d_lr: torch.Tensor, stream=None):
        B.lars_step(self.handle, hyper,
                    d_step.data_ptr() if d_step is not None else 0,
                    d_lr.data_ptr(), _stream(stream))

    def nlamb_step(self, hyper, momentum_decay, nesterov_second_moment,
                   d_step: torch.Tensor, d_lr: torch.Tensor,
                   d_mu_product: torch.Tensor, stream=None):
        B.nlamb_step(self.handle, hyper, momentum_decay,
                     nesterov_second_moment, d_step.data_ptr(),
                     d_lr.data_ptr(), d_mu_product.data_ptr(),
                     _stream(stream))

    def step_call(self, kind, hyper, d_step: torch.Tensor, d_lr: torch.Tensor,
                  d_mu_product: torch.Tensor = None, momentum_decay=0.004,
                  stream=None):
        """binding.step_call on this plan: a zero-argument callable for one
        step, with the device pointers and the stream taken now."""
        return B.step_call(kind, self.handle, hyper,
                           d_step.data_ptr() if d_step is not None else 0,
                           d_lr.data_ptr(), _stream(stream), momentum_decay,
                           d_mu_product.data_ptr()
                           if d_mu_product is not None else 0)

    def results(self, stream=None):
        """(ratio, wnorm, unorm) as new float64 device tensors."""
        dev = self.state.device
        out = [torch.empty(self.n, dtype=torch.float64, device=dev)
               for _ in range(3)]
        B.lamb_plan_copy_trust_ratios(self.handle, *(t.data_ptr() for t in out),
                                      stream=_stream(stream))
        return out

    def grad_norms(self, stream=None):
        """(||g_k|| [n] f64, global ||g|| [1] f64, non-finite flag [1] i32)
        of the last step with the gradient check, as new device tensors."""
        dev = self.state.device
        out = (torch.empty(self.n, dtype=torch.float64, device=dev),
               torch.empty(1, dtype=torch.float64, device=dev),
               torch.empty(1, dtype=torch.int32, device=dev))
        B.lamb_plan_copy_grad_norms(self.handle, *(t.data_ptr() for t in out),
                                    stream=_stream(stream))
        return out

    # -- sharded step (data-parallel) -------------------------------------
    def shard_pass1(self, hyper, optimizer, d_step, d_lr, d_mu_product=None,
                    momentum_decay=0.0, stream=None):
        B.lamb_shard_pass1(self.handle, hyper, optimizer, momentum_decay,
                           d_step.data_ptr() if d_step is not None else 0,
                           d_lr.data_ptr() if d_lr is not None else 0,
                           d_mu_product.data_ptr()
                           if d_mu_product is not None else 0, _stream(stream))

    def shard_pass2(self, hyper, optimizer, d_step, d_lr, d_mu_product=None,
                    momentum_decay=0.0, stream=None):
        B.lamb_shard_pass2(self.handle, hyper, optimizer, momentum_decay,
                           d_step.data_ptr() if d_step is not None else 0,
                           d_lr.data_ptr() if d_lr is not None else 0,
                           d_mu_product.data_ptr()
                           if d_mu_product is not None else 0, _stream(stream))

    def partials(self, stream=None) -> torch.Tensor:
        """A device copy of the per-chunk sums (for an all-reduce)."""
        _, n = B.lamb_plan_partials(self.handle)
        out = torch.empty(n, dtype=torch.float32, device=self.state.device)
        B.lamb_plan_copy_partials(self.handle, out.data_ptr(), False,
                                  _stream(stream))
        return out

    def set_partials(self, t: torch.Tensor, stream=None) -> None:
        """Put the (all-reduced) per-chunk sums back into the plan."""
        _, n = B.lamb_plan_partials(self.handle)
        assert t.dtype == torch.float32 and t.numel() == n and t.is_contiguous()
        B.lamb_plan_copy_partials(self.handle, t.data_ptr(), True,
                                  _stream(stream))

    def query(self, clear=False, stream=None) -> int:
        return B.lamb_plan_query(self.handle, clear, _stream(stream))

    def info(self) -> dict:
        return B.lamb_plan_get_info(self.handle)

    def destroy(self):
        if self.handle:
            B.lamb_plan_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass


def _stream(stream):
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream
