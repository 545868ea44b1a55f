"""Pins for the oracle's gradient check (reading Q17) and decoupled weight
decay (reading Q18), against things other than the oracle itself: integer
vectors whose norms are integers, closed forms, exact rational sums of the
fp32 inputs, IEEE special values, torch's AdamW / NAdam with decoupled
decay, and planted mistakes that these pins must reject."""
import inspect
import math
from fractions import Fraction

import numpy as np
import pytest

from oracle import lamb_oracle as O


# ---------------------------------------------------------------------------
# Gradient norms (Q17)
# ---------------------------------------------------------------------------

def _f32(*x):
    return np.array(x, dtype=np.float32)


def test_grad_norms_of_pythagorean_blocks():
    # (3, 4) -> 5, (12) -> 12, whole gradient (3, 4, 12) -> 13
    r = O.grad_check([_f32(3, 4), _f32(12)])
    assert r.norms == [5.0, 12.0] and r.norm == 13.0 and not r.nonfinite
    # (2, 3, 6) -> 7 split over three blocks, one of them empty
    r = O.grad_check([_f32(2), _f32(), _f32(-3, 6)])
    assert r.norms == [2.0, 0.0, math.sqrt(45.0)] and r.norm == 7.0


def test_grad_norms_of_bf16_patterns():
    # bf16 3.0 = 0x4040, -4.0 = 0xC080: the patterns are the top halves of
    # the fp32 values
    r = O.grad_check([np.array([0x4040, 0xC080], dtype=np.uint16)],
                     g_dtype="bf16")
    assert r.norms == [5.0] and r.norm == 5.0


@pytest.mark.parametrize("blocks", [[(0.5, 16)], [(0.25, 64), (3.0, 1)],
                                    [(1e-3, 1000), (2.0, 4), (-7.0, 9)]])
def test_grad_norms_of_constant_blocks(blocks):
    # a block of n copies of c has norm |c| sqrt(n)
    gs = [np.full(n, c, dtype=np.float32) for c, n in blocks]
    r = O.grad_check(gs)
    for got, (c, n) in zip(r.norms, blocks):
        cf = float(np.float32(c))
        assert math.isclose(got, abs(cf) * math.sqrt(n), rel_tol=1e-15)
    want = math.sqrt(sum(float(np.float32(c)) ** 2 * n for c, n in blocks))
    assert math.isclose(r.norm, want, rel_tol=1e-15)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_grad_norms_match_exact_rational_sum(seed):
    rng = np.random.default_rng(seed)
    gs = [rng.normal(0, 10.0 ** rng.integers(-6, 2), rng.integers(1, 40))
          .astype(np.float32) for _ in range(5)]
    r = O.grad_check(gs)
    exact = [sum(Fraction(float(x)) ** 2 for x in g) for g in gs]
    for got, e in zip(r.norms, exact):
        assert math.isclose(got, math.sqrt(float(e)), rel_tol=4e-16)
    assert math.isclose(r.norm, math.sqrt(float(sum(exact))), rel_tol=4e-16)


def test_grad_norm_is_invariant_to_blocking_and_order():
    rng = np.random.default_rng(5)
    g = rng.normal(0, 1e-2, 1000).astype(np.float32)
    whole = O.grad_check([g]).norm
    parts = O.grad_check([g[:7], g[7:500], g[500:][::-1]]).norm
    assert math.isclose(whole, parts, rel_tol=1e-15)


@pytest.mark.parametrize("bad", [np.inf, -np.inf, np.nan])
@pytest.mark.parametrize("where", [0, 5, -1])
def test_nonfinite_element_is_detected_anywhere(bad, where):
    gs = [np.ones(3, np.float32), np.ones(8, np.float32), np.ones(2, np.float32)]
    gs[1][where] = bad
    r = O.grad_check(gs)
    assert r.nonfinite
    assert not math.isfinite(r.norms[1]) and not math.isfinite(r.norm)
    assert math.isfinite(r.norms[0]) and math.isfinite(r.norms[2])


def test_extreme_finite_values_are_not_nonfinite():
    fmax = np.finfo(np.float32).max
    tiny = np.float32(1e-45)                    # smallest fp32 denormal
    r = O.grad_check([_f32(fmax, -fmax), _f32(tiny, -0.0, 0.0)])
    assert not r.nonfinite
    # fmax^2 overflows fp32 but not float64
    assert math.isclose(r.norms[0], float(fmax) * math.sqrt(2), rel_tol=1e-15)
    assert r.norms[1] == float(tiny)
    bits = np.array([0x7F7F, 0x0001, 0x8000], dtype=np.uint16)  # bf16 max, denormal, -0
    assert not O.grad_check([bits], g_dtype="bf16").nonfinite
    inf_bits = np.array([0x3F80, 0x7F80], dtype=np.uint16)       # 1.0, +Inf
    assert O.grad_check([inf_bits], g_dtype="bf16").nonfinite


def _grad_mutant(kind):
    def check(gs, g_dtype="f32"):
        sq, bad = [], False
        for g in gs:
            x = O.to_f64(g, g_dtype)
            if kind == "nan_missed":
                bad |= bool(np.any(np.isinf(x)))
            else:
                bad |= not bool(np.all(np.isfinite(x)))
            sq.append(float(np.sum(np.abs(x))) if kind == "no_square"
                      else float(np.sum(x * x)))
        norms = [math.sqrt(s) for s in sq]
        total = (sum(norms) if kind == "sum_of_norms" else
                 math.sqrt(sum(sq)))
        return O.GradCheck(norms, total, bad)
    return check


@pytest.mark.parametrize("kind", ["no_square", "sum_of_norms", "nan_missed"])
def test_grad_pins_reject_planted_mistake(kind, monkeypatch):
    monkeypatch.setattr(O, "grad_check", _grad_mutant(kind))
    failed = 0
    for pin in (test_grad_norms_of_pythagorean_blocks,
                lambda: test_nonfinite_element_is_detected_anywhere(np.nan, 0)):
        try:
            pin()
        except AssertionError:
            failed += 1
    assert failed, f"planted mistake {kind!r} passed the pins"


# ---------------------------------------------------------------------------
# Decoupled weight decay (Q18)
# ---------------------------------------------------------------------------

def _block(rng, n, warm=True):
    w = rng.normal(0, 0.02, n)
    g = rng.normal(0, 1e-3, n)
    m = rng.normal(0, 3e-4, n) if warm else np.zeros(n)
    v = 1e-6 * rng.uniform(0.0005, 0.003, n) if warm else np.zeros(n)
    return w, g, m, v


@pytest.mark.parametrize("phi_kind,gu", [("identity", math.inf),
                                         ("clip", 1e-3)])
def test_decoupled_step_norm_closed_form(phi_kind, gu):
    # x' - x + lr*lam*x is the normalised step: its norm is lr * phi(||x||)
    rng = np.random.default_rng(11)
    w, g, m, v = _block(rng, 257)
    lr, wd = 3e-3, 0.05
    res = O.lamb_tensor(w, g, m, v, t=7, lr=lr, weight_decay=wd,
                        decoupled_decay=True, phi_kind=phi_kind, gamma_u=gu)
    step = res.w - w + lr * wd * w
    want = lr * min(np.linalg.norm(w), gu)
    # the subtraction cancels: its rounding is relative to |w|, not the step
    tol = 8 * np.finfo(float).eps * np.linalg.norm(w) / want
    assert math.isclose(np.linalg.norm(step), want, rel_tol=tol)


def test_decoupled_equals_coupled_without_decay():
    rng = np.random.default_rng(12)
    w, g, m, v = _block(rng, 100)
    for kw in (dict(weight_decay=0.0), dict(weight_decay=0.1, decay=False)):
        a = O.lamb_tensor(w, g, m, v, t=3, lr=1e-3, decoupled_decay=True, **kw)
        b = O.lamb_tensor(w, g, m, v, t=3, lr=1e-3, **kw)
        np.testing.assert_array_equal(a.w, b.w)
        assert a.ratio == b.ratio


torch = pytest.importorskip("torch")


def _torch_step(opt_cls, w, g, m, v, t, **kw):
    p = torch.tensor(w, dtype=torch.float64, requires_grad=True)
    opt = opt_cls([p], **kw)
    state = {"step": torch.tensor(float(t - 1), dtype=torch.float64),
             "exp_avg": torch.tensor(m, dtype=torch.float64),
             "exp_avg_sq": torch.tensor(v, dtype=torch.float64)}
    opt.state[p] = state
    p.grad = torch.tensor(g, dtype=torch.float64)
    opt.step()
    return p.detach().numpy()


@pytest.mark.parametrize("t", [1, 5])
def test_decoupled_lamb_with_unit_ratio_is_torch_adamw(t):
    # With phi clipped to the constant ||r|| the trust ratio is 1 and the
    # decoupled LAMB step is AdamW's: x - lr*r - lr*lam*x.  ||r|| comes from
    # torch's Adam (lr = 1, no decay: its step is exactly -r).
    rng = np.random.default_rng(20 + t)
    w, g, m, v = _block(rng, 64, warm=t > 1)
    r = w - _torch_step(torch.optim.Adam, w, g, m, v, t, lr=1.0,
                        betas=(0.9, 0.999), eps=1e-6)
    rn = float(np.linalg.norm(r))
    lr, wd = 2e-3, 0.01
    want = _torch_step(torch.optim.AdamW, w, g, m, v, t, lr=lr,
                       betas=(0.9, 0.999), eps=1e-6, weight_decay=wd)
    res = O.lamb_tensor(w, g, m, v, t=t, lr=lr, weight_decay=wd,
                        decoupled_decay=True, phi_kind="clip", gamma_l=rn,
                        gamma_u=rn)
    np.testing.assert_allclose(res.w, want, rtol=1e-13, atol=1e-19)
    assert math.isclose(res.ratio, 1.0, rel_tol=1e-13)


def test_decoupled_nlamb_with_unit_ratio_is_torch_nadam():
    if "decoupled_weight_decay" not in inspect.signature(
            torch.optim.NAdam).parameters:
        pytest.skip("torch NAdam without decoupled_weight_decay")
    rng = np.random.default_rng(31)
    w, g, m, v = _block(rng, 48)
    t, psi, b1 = 4, 0.004, 0.975
    mu_prev = math.prod(O.nadam_mu(i, b1, psi) for i in range(1, t))

    def nadam(lr, wd):
        p = torch.tensor(w, dtype=torch.float64, requires_grad=True)
        opt = torch.optim.NAdam([p], lr=lr, betas=(b1, 0.999), eps=1e-8,
                                weight_decay=wd, momentum_decay=psi,
                                decoupled_weight_decay=True)
        opt.state[p] = {"step": torch.tensor(float(t - 1), dtype=torch.float64),
                        "mu_product": torch.tensor(mu_prev, dtype=torch.float64),
                        "exp_avg": torch.tensor(m, dtype=torch.float64),
                        "exp_avg_sq": torch.tensor(v, dtype=torch.float64)}
        p.grad = torch.tensor(g, dtype=torch.float64)
        opt.step()
        return p.detach().numpy()

    r = w - nadam(1.0, 0.0)
    rn = float(np.linalg.norm(r))
    lr, wd = 1e-3, 0.02
    want = nadam(lr, wd)
    res = O.nlamb_tensor(w, g, m, v, t=t, lr=lr, mu_product=mu_prev,
                         beta1=b1, psi=psi, weight_decay=wd,
                         decoupled_decay=True, phi_kind="clip", gamma_l=rn,
                         gamma_u=rn)
    np.testing.assert_allclose(res.w, want, rtol=1e-12, atol=1e-19)


def _decoupled_mutant(kind):
    real = O.lamb_tensor

    def lamb(w, g, m, v, *, decoupled_decay=False, **kw):
        if not decoupled_decay:
            return real(w, g, m, v, **kw)
        res = real(w, g, m, v, decoupled_decay=False, **kw)
        if kind == "coupled":
            return res
        # decay scaled by the trust ratio instead of by lr alone
        lam = kw.get("weight_decay", 0.01) if kw.get("decay", True) else 0.0
        base = real(w, g, m, v, weight_decay=0.0,
                    **{k: x for k, x in kw.items() if k != "weight_decay"})
        x = O.to_f64(w)
        return O.LambResult(base.w - kw["lr"] * base.ratio * lam * x, base.m,
                            base.v, base.ratio, base.wnorm, base.unorm)
    return lamb


@pytest.mark.parametrize("kind", ["coupled", "decay_times_ratio"])
def test_decoupled_pins_reject_planted_mistake(kind, monkeypatch):
    monkeypatch.setattr(O, "lamb_tensor", _decoupled_mutant(kind))
    failed = 0
    for pin in (lambda: test_decoupled_lamb_with_unit_ratio_is_torch_adamw(5),
                lambda: test_decoupled_step_norm_closed_form("identity",
                                                             math.inf)):
        try:
            pin()
        except AssertionError:
            failed += 1
    assert failed, f"planted mistake {kind!r} passed the pins"
