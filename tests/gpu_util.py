"""Helpers for the GPU parity tests: load layouts onto the device, run the
CUDA path through the C ABI, run the fp64 oracle on the same inputs, and
compare element by element.

Tolerances (per element, |gpu - ref| <= tol * scale):
  w: scale = max(|ref|, |w_old|)       (the update is small next to w);
     along a chain also the element's oracle path sum_t |w_t - w_{t-1}|:
     each step's error is relative to that step's update, so near a zero
     crossing |w| alone says nothing about the accumulated error
     and the update's size built from its operands' magnitudes,
     lr*rho*(c1*(beta1|m_old| + (1-beta1)|g|)/(sqrt(v_hat)+eps) + lambda|w|)
     (LARS: lr*rho*(beta1|m_old| + (1-beta1)(|g| + lambda|w|))): when m
     cancels and w is 0 the update's error follows its operands
  m: scale = max(|ref|, |beta1 m_old| + |(1-beta1) g|  [+ lambda |w| LARS])
     fp32 error follows the operands, not a cancelled result; along a chain
     the running operand size M_t = beta1 M_{t-1} + (1-beta1)|g_t| [+...]
     (earlier steps' rounding is carried forward with factor beta1)
  v: scale = |ref|                     (a sum of non-negative terms)
  trust ratio: relative 1e-6
tol = 1e-5 after one step, 1e-4 along chained runs.
"""
from __future__ import annotations

import math
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import torch

from oracle import lamb_oracle as O
from paper_1904_00962_gb300 import binding as B
from paper_1904_00962_gb300.state import DeviceState, LambPlan

# the step algorithms of the library
ALGOS = [1, 3]
ALGO_IDS = {1: "two_pass", 3: "on_chip"}

TOL_STEP = 1e-5
TOL_CHAIN = 1e-4
TOL_RATIO = 1e-6


def hyper_kwargs(h, lars=False):
    """Oracle keyword arguments of a workloads.Hyper."""
    kw = dict(beta1=h.beta1, weight_decay=h.weight_decay, phi_kind=h.phi,
              gamma_l=h.gamma_l, gamma_u=h.gamma_u)
    if lars:
        kw["trust_coef"] = h.trust_coef
    else:
        kw.update(beta2=h.beta2, eps=h.eps, bias_correction=h.bias_correction)
    return kw


def c_hyper(h, lars=False, increment=False):
    return B.make_hyper(beta1=h.beta1, beta2=h.beta2, eps=h.eps,
                        weight_decay=h.weight_decay, phi=h.phi,
                        gamma_l=h.gamma_l, gamma_u=h.gamma_u,
                        trust_coef=h.trust_coef,
                        bias_correction=(h.bias_correction and not lars),
                        increment_step=increment)


def f32(x):
    return float(np.float32(x))


def _nan_aware_ok(err, bound, got, ref):
    both_nan = np.isnan(got) & np.isnan(ref)
    return np.all((err <= bound) | both_nan)


# How often the tolerance floors decide a comparison: per test, the elements
# compared, those whose error exceeds tol * |ref| but not tol * floor (they
# pass only because of a floor), and the worst plain relative error
# |gpu - ref| / |ref|.  Written out by conftest when LAMB_FLOOR_STATS names a
# file.
FLOOR_STATS = {}


def _floor_stat(array, err, ref, scale, tol):
    import os
    test = os.environ.get("PYTEST_CURRENT_TEST", "?").split(" ")[0]
    ref = np.abs(ref)
    fin = np.isfinite(err) & np.isfinite(ref)
    floored = fin & (err > tol * ref) & (err <= tol * scale)
    with np.errstate(divide="ignore", invalid="ignore"):
        rel = np.where(fin & (ref > 0), err / np.where(ref > 0, ref, 1.0), 0.0)
    st = FLOOR_STATS.setdefault(test, {})
    a = st.setdefault(array, {"n": 0, "floored": 0, "worst_plain_rel": 0.0,
                              "tol": tol})
    a["n"] += int(err.size)
    a["floored"] += int(floored.sum())
    if rel.size:
        a["worst_plain_rel"] = max(a["worst_plain_rel"], float(np.max(rel)))


def rel_max(err, scale):
    with np.errstate(divide="ignore", invalid="ignore"):
        r = np.where(scale > 0, err / scale, np.where(err > 0, np.inf, 0.0))
    r = r[~np.isnan(r)]
    return float(r.max()) if r.size else 0.0


def compare_lamb(got_w, got_m, got_v, ref, w_old, m_old, g64, beta1, tol,
                 w_path=None, upd=None, m_path=None):
    """Returns dict of max scaled errors; raises AssertionError on failure.
    upd = (hyper, t, lr, lam) enables the update-operand floor of w."""
    got_w = got_w.astype(np.float64)
    got_m = got_m.astype(np.float64)
    m_op = beta1 * np.abs(m_old) + (1 - beta1) * np.abs(g64)
    sw = np.maximum(np.abs(ref.w), np.abs(w_old))
    if w_path is not None:
        sw = np.maximum(sw, w_path)
    if upd is not None:
        h, t, lr, lam = upd
        c1 = 1 / (1 - h.beta1 ** t) if h.bias_correction else 1.0
        c2 = 1 / (1 - h.beta2 ** t) if h.bias_correction else 1.0
        u_op = c1 * m_op / (np.sqrt(ref.v * c2) + h.eps) + lam * np.abs(w_old)
        if np.isfinite(ref.ratio):
            sw = np.maximum(sw, lr * ref.ratio * u_op)
    sm = np.maximum(np.abs(ref.m), m_op)
    if m_path is not None:
        sm = np.maximum(sm, m_path)
    ew, em = np.abs(got_w - ref.w), np.abs(got_m - ref.m)
    assert _nan_aware_ok(ew, tol * sw, got_w, ref.w), f"w err {rel_max(ew, sw)}"
    assert _nan_aware_ok(em, tol * sm, got_m, ref.m), f"m err {rel_max(em, sm)}"
    _floor_stat("w", ew, ref.w, sw, tol)
    _floor_stat("m", em, ref.m, sm, tol)
    out = {"w": rel_max(ew, sw), "m": rel_max(em, sm), "_sw": sw}
    if got_v is not None:
        got_v = got_v.astype(np.float64)
        ev, sv = np.abs(got_v - ref.v), np.abs(ref.v)
        assert _nan_aware_ok(ev, tol * sv, got_v, ref.v), f"v err {rel_max(ev, sv)}"
        out["v"] = rel_max(ev, sv)
    return out


def compare_lars(got_w, got_m, ref, w_old, m_old, g64, beta1, lam, tol,
                 w_path=None, lr=None, m_path=None):
    """lr enables the update-operand floor of w."""
    got_w = got_w.astype(np.float64)
    got_m = got_m.astype(np.float64)
    m_op = beta1 * np.abs(m_old) + (1 - beta1) * (np.abs(g64) +
                                                  lam * np.abs(w_old))
    sw = np.maximum(np.abs(ref.w), np.abs(w_old))
    if w_path is not None:
        sw = np.maximum(sw, w_path)
    if lr is not None and np.isfinite(ref.ratio):
        sw = np.maximum(sw, lr * ref.ratio * m_op)
    sm = np.maximum(np.abs(ref.m), m_op)
    if m_path is not None:
        sm = np.maximum(sm, m_path)
    ew, em = np.abs(got_w - ref.w), np.abs(got_m - ref.m)
    assert _nan_aware_ok(ew, tol * sw, got_w, ref.w), f"w err {rel_max(ew, sw)}"
    assert _nan_aware_ok(em, tol * sm, got_m, ref.m), f"m err {rel_max(em, sm)}"
    _floor_stat("w", ew, ref.w, sw, tol)
    _floor_stat("m", em, ref.m, sm, tol)
    return {"w": rel_max(ew, sw), "m": rel_max(em, sm), "_sw": sw}


def compare_nlamb(got_w, got_m, got_v, ref, w_old, m_old, g64, h, t, lr, lam,
                  psi, mu_product, nn, tol, w_path=None, m_path=None):
    """compare_lamb for N-LAMB / NN-LAMB (appendix Algs. 3/4): the same
    floors, with the update-operand floor built from the Nesterov form."""
    from oracle import lamb_oracle as O
    mu_t = O.nadam_mu(t, h.beta1, psi)
    mu_n = O.nadam_mu(t + 1, h.beta1, psi)
    p_t = mu_product * mu_t
    am, ag = mu_n / (1 - p_t * mu_n), (1 - mu_t) / (1 - p_t)
    if nn:
        vh = (h.beta2 * ref.v / (1 - h.beta2 ** (t + 1))
              + (1 - h.beta2) * g64 * g64 / (1 - h.beta2 ** t))
    else:
        vh = ref.v / (1 - h.beta2 ** t)
    m_op = h.beta1 * np.abs(m_old) + (1 - h.beta1) * np.abs(g64)
    u_op = (am * m_op + ag * np.abs(g64)) / (np.sqrt(vh) + h.eps) + \
        lam * np.abs(w_old)
    got_w = got_w.astype(np.float64)
    got_m = got_m.astype(np.float64)
    got_v = got_v.astype(np.float64)
    sw = np.maximum(np.abs(ref.w), np.abs(w_old))
    if w_path is not None:
        sw = np.maximum(sw, w_path)
    if np.isfinite(ref.ratio):
        sw = np.maximum(sw, lr * ref.ratio * u_op)
    sm = np.maximum(np.abs(ref.m), m_op)
    if m_path is not None:
        sm = np.maximum(sm, m_path)
    ew, em, ev = (np.abs(got_w - ref.w), np.abs(got_m - ref.m),
                  np.abs(got_v - ref.v))
    assert _nan_aware_ok(ew, tol * sw, got_w, ref.w), f"w err {rel_max(ew, sw)}"
    assert _nan_aware_ok(em, tol * sm, got_m, ref.m), f"m err {rel_max(em, sm)}"
    assert _nan_aware_ok(ev, tol * np.abs(ref.v), got_v, ref.v), \
        f"v err {rel_max(ev, np.abs(ref.v))}"
    _floor_stat("w", ew, ref.w, sw, tol)
    _floor_stat("m", em, ref.m, sm, tol)
    return {"w": rel_max(ew, sw), "m": rel_max(em, sm), "_sw": sw}


def worst_of(errs):
    return max(v for k, v in errs.items() if not k.startswith("_"))


def ratio_ok(got, want, tol=TOL_RATIO):
    if math.isnan(want):
        return math.isnan(got)
    return abs(got - want) <= tol * abs(want)


def _bf16_ordered(bits):
    b = bits.astype(np.int32)
    return np.where(b & 0x8000, -(b & 0x7FFF), b)


def check_copy(copy_bits, got_w32, ref_w64, sw=None, tol=TOL_STEP):
    """bf16 copy == RNE(gpu fp32 w) bit-exactly, and within 1 bf16 ulp of
    RNE(oracle w rounded to fp32) -- or, where the w comparison needed its
    floors (sw > |ref|), within half a bf16 ulp of ref plus tol*sw, which is
    what the two other checks together imply."""
    np.testing.assert_array_equal(copy_bits, O.bf16_rne(got_w32))
    want = _bf16_ordered(O.bf16_rne(ref_w64.astype(np.float32)))
    got = _bf16_ordered(copy_bits)
    ok = np.abs(got - want) <= 1
    if sw is not None and not ok.all():
        val = O.bf16_bits_to_f64(copy_bits)
        ok |= np.abs(val - ref_w64) <= 2.0 ** -8 * np.abs(ref_w64) + tol * sw
    assert np.all(ok)


class GpuLayout:
    """A layout's state on the GPU plus a bound plan."""

    def __init__(self, layout, *, with_v=True, chunk_elems=0, blocks_per_sm=0,
                 misalign=None, device="cuda:0", algorithm=1, **plan_opts):
        self.L = layout
        self.st = DeviceState(layout.sizes, grad_dtype=layout.grad_dtype,
                              copy_dtype=layout.copy_dtype, device=device,
                              with_v=with_v, misalign=misalign)
        self.plan = LambPlan(self.st, layout.decay, chunk_elems=chunk_elems,
                             blocks_per_sm=blocks_per_sm, algorithm=algorithm,
                             **plan_opts)
        self.d_step = torch.ones(1, dtype=torch.int64, device=device)
        self.d_lr = torch.zeros(1, dtype=torch.float32, device=device)

    def load_weights(self, ks=None):
        for k in (range(self.L.n_tensors) if ks is None else ks):
            self.st.upload("w", k, self.L.weights(k))

    def load_grads(self, step, ks=None):
        for k in (range(self.L.n_tensors) if ks is None else ks):
            self.st.upload("g", k, self.L.grad(k, step))

    def load_warm_state(self, ks=None):
        for k in (range(self.L.n_tensors) if ks is None else ks):
            m, v = self.L.state_warm(k)
            self.st.upload("m", k, m)
            if self.st.v is not None:
                self.st.upload("v", k, v)

    def step(self, t, lr, hyper, lars=False):
        self.d_step.fill_(int(t))
        self.d_lr.fill_(float(lr))
        if lars:
            self.plan.lars_step(hyper, self.d_step, self.d_lr)
        else:
            self.plan.lamb_step(hyper, self.d_step, self.d_lr)

    def results(self, check_status=True):
        """Trust ratios and norms of the last step; by default also asserts
        that the device status word is clear (no non-finite norm, bad step
        count or abandoned wait)."""
        r, w, u = self.plan.results()
        torch.cuda.synchronize()
        if check_status:
            st = self.plan.query()
            assert st == 0, f"device status 0x{st:x}"
        return r.cpu().numpy(), w.cpu().numpy(), u.cpu().numpy()

    def download(self, name, k):
        return self.st.download(name, k)

    def close(self):
        self.plan.destroy()


def oracle_map(fn, items, workers=8):
    """Runs fn over items with a thread pool (NumPy releases the GIL in its
    large array operations)."""
    with ThreadPoolExecutor(workers) as ex:
        return list(ex.map(fn, items))
