"""Pins for the N-LAMB / NN-LAMB oracle (appendix Algorithms 3 and 4):
hand-derived exact cases, torch's NAdam (Dozat's Nadam, with decoupled
weight decay) as the library special case of N-LAMB's direction, the sign-SGD
reduction, the step-norm closed form and the momentum-product recurrence,
plus planted mistakes the pins must reject."""
import json
import math
import os

import numpy as np
import pytest
import sympy

from oracle import lamb_oracle as O

HERE = os.path.dirname(os.path.abspath(__file__))
GOLDEN = os.path.join(HERE, "golden", "nlamb_hand_cases.json")


def _ev(expr):
    return float(sympy.N(sympy.sympify(expr), 40))


def _cases():
    with open(GOLDEN) as f:
        return json.load(f)["cases"]


def _run(case, fn=None):
    fn = fn or O.nlamb_tensor
    h = case["hyper"]
    arr = lambda k: np.array([_ev(s) for s in case[k]])
    return fn(arr("w"), arr("g"), arr("m"), arr("v"), t=h["t"],
              lr=_ev(h["lr"]), mu_product=_ev(h["mu_product"]),
              beta1=_ev(h["beta1"]), beta2=_ev(h["beta2"]), eps=_ev(h["eps"]),
              psi=_ev(h["psi"]), weight_decay=_ev(h["weight_decay"]),
              decay=h["decay"],
              nesterov_second_moment=case["nesterov_second_moment"])


def _matches(case, res, rtol=1e-12):
    exp = case["expected"]
    ok = True
    for key in ("w", "m", "v"):
        ok &= np.allclose(getattr(res, key), [_ev(s) for s in exp[key]],
                          rtol=rtol, atol=1e-15)
    for key in ("ratio", "wnorm", "unorm", "mu_product"):
        ok &= math.isclose(getattr(res, key), _ev(exp[key]), rel_tol=rtol,
                           abs_tol=1e-15)
    return bool(ok)


@pytest.mark.parametrize("case", _cases(), ids=lambda c: c["name"])
def test_hand_case(case):
    res = _run(case)
    exp = case["expected"]
    for key in ("w", "m", "v"):
        np.testing.assert_allclose(getattr(res, key),
                                   [_ev(s) for s in exp[key]], rtol=1e-12,
                                   atol=1e-15, err_msg=key)
    for key in ("ratio", "wnorm", "unorm", "mu_product"):
        assert math.isclose(getattr(res, key), _ev(exp[key]), rel_tol=1e-12,
                            abs_tol=1e-15), key


def _block(rng, n, warm=True):
    w = rng.normal(0, 0.02, n)
    g = rng.normal(0, 1e-3, n)
    m = rng.normal(0, 3e-4, n) if warm else np.zeros(n)
    v = 1e-6 * rng.uniform(5e-4, 3e-3, n) if warm else np.zeros(n)
    return w, g, m, v


# ---------------------------------------------------------------------------
# Library special case: Algorithm 3's m_hat/(sqrt(v_hat)+eps) + lambda*x is
# the per-element update of Dozat's Nadam with decoupled weight decay at
# learning rate 1 (torch.optim.NAdam, same schedule and product state).
# ---------------------------------------------------------------------------

torch = pytest.importorskip("torch")


def _nadam_direction(w, g, m, v, t, mu_product, beta1, beta2, eps, psi, wd):
    p = torch.tensor(w, dtype=torch.float64, requires_grad=True)
    opt = torch.optim.NAdam([p], lr=1.0, betas=(beta1, beta2), eps=eps,
                            weight_decay=wd, momentum_decay=psi,
                            decoupled_weight_decay=True)
    opt.state[p] = {"step": torch.tensor(float(t - 1), dtype=torch.float64),
                    "mu_product": torch.tensor(mu_product, dtype=torch.float64),
                    "exp_avg": torch.tensor(m, dtype=torch.float64),
                    "exp_avg_sq": torch.tensor(v, dtype=torch.float64)}
    p.grad = torch.tensor(g, dtype=torch.float64)
    opt.step()
    st = opt.state[p]
    return (w - p.detach().numpy(), st["exp_avg"].numpy(),
            st["exp_avg_sq"].numpy(), float(st["mu_product"]))


@pytest.mark.parametrize("t", [1, 2, 37, 1000])
@pytest.mark.parametrize("decay", [True, False])
@pytest.mark.parametrize("psi", [0.004, 0.0])
def test_nlamb_direction_is_nadam_update(t, decay, psi):
    rng = np.random.default_rng(t * 7 + decay)
    n = 211
    w, g, m, v = _block(rng, n, warm=t > 1)
    beta1, beta2, eps = 0.975, 0.999, 1e-8
    prod = 1.0
    for i in range(1, t):
        prod *= O.nadam_mu(i, beta1, psi)
    wd = 0.01
    u, m_t, v_t, prod_t = _nadam_direction(w, g, m, v, t, prod, beta1, beta2,
                                           eps, psi, wd if decay else 0.0)
    lr = 2e-3
    res = O.nlamb_tensor(w, g, m, v, t=t, lr=lr, mu_product=prod,
                         beta1=beta1, beta2=beta2, eps=eps, psi=psi,
                         weight_decay=wd, decay=decay)
    scale = beta1 * np.abs(m) + (1 - beta1) * np.abs(g)
    assert np.all(np.abs(res.m - m_t) <= 1e-14 * np.maximum(scale, np.abs(m_t)))
    np.testing.assert_allclose(res.v, v_t, rtol=1e-14, atol=0)
    assert math.isclose(res.mu_product, prod_t, rel_tol=1e-14)
    assert math.isclose(res.unorm, np.linalg.norm(u), rel_tol=1e-10)
    want = w - lr * np.linalg.norm(w) / np.linalg.norm(u) * u
    np.testing.assert_allclose(res.w, want, rtol=1e-12, atol=1e-18)


def test_momentum_product_recurrence():
    beta1, psi = 0.975, 0.004
    rng = np.random.default_rng(1)
    w, g, m, v = _block(rng, 17, warm=False)
    prod = 1.0
    for t in range(1, 30):
        r = O.nlamb_tensor(w, g, m, v, t=t, lr=1e-3, mu_product=prod,
                           beta1=beta1, psi=psi)
        prod, w, m, v = r.mu_product, r.w, r.m, r.v
    want = math.prod(beta1 * (1 - 0.5 * 0.96 ** (i * psi)) for i in range(1, 30))
    assert math.isclose(prod, want, rel_tol=1e-14)


@pytest.mark.parametrize("nn", [False, True])
def test_step_norm_closed_form(nn):
    rng = np.random.default_rng(3)
    w, g, m, v = _block(rng, 999)
    res = O.nlamb_tensor(w, g, m, v, t=5, lr=3e-3, mu_product=0.5,
                         nesterov_second_moment=nn, phi_kind="clip",
                         gamma_u=0.1)
    assert math.isclose(np.linalg.norm(res.w - w), 3e-3 * 0.1, rel_tol=1e-9)


def test_nnlamb_sign_sgd_reduction():
    """beta1 = beta2 = 0: mu_t = 0, m_hat = g and (NN-LAMB) v_hat = g^2, so
    r = sign(g) and the step is sign-SGD scaled by sqrt(d) (cf. the remark
    under Algorithm 2)."""
    rng = np.random.default_rng(4)
    w, g, m, v = _block(rng, 500)
    res = O.nlamb_tensor(w, g, m, v, t=3, lr=1e-2, mu_product=0.3, beta1=0.0,
                         beta2=0.0, eps=1e-300, weight_decay=0.0,
                         nesterov_second_moment=True)
    assert math.isclose(res.unorm, math.sqrt(500), rel_tol=1e-12)
    want = w - 1e-2 * np.linalg.norm(w) / math.sqrt(500) * np.sign(g)
    np.testing.assert_allclose(res.w, want, rtol=1e-12, atol=1e-18)


def test_rejects_bad_step():
    with pytest.raises(ValueError):
        O.nlamb_tensor(np.ones(2), np.ones(2), np.zeros(2), np.zeros(2), t=0,
                       lr=1e-3, mu_product=1.0)


# ---------------------------------------------------------------------------
# Planted mistakes
# ---------------------------------------------------------------------------

def _mutant(kind):
    def fn(w, g, m, v, *, t, lr, mu_product, beta1=0.975, beta2=0.999,
           eps=1e-8, psi=0.004, weight_decay=0.01, decay=True,
           nesterov_second_moment=False, **kw):
        x, gt = np.asarray(w, float), np.asarray(g, float)
        lam = weight_decay if decay else 0.0
        mu_t, mu_n = O.nadam_mu(t, beta1, psi), O.nadam_mu(t + 1, beta1, psi)
        if kind == "schedule_as_power":
            mu_t, mu_n = beta1 ** t, beta1 ** (t + 1)
        p_t = mu_product * mu_t
        p_n = p_t * mu_n
        if kind == "product_off_by_one":
            p_n = p_t
        m_t = beta1 * np.asarray(m, float) + (1 - beta1) * gt
        m_hat = mu_n * m_t / (1 - p_n) + (1 - mu_t) * gt / (1 - p_t)
        if kind == "no_gradient_term":
            m_hat = mu_n * m_t / (1 - p_n)
        v_t = beta2 * np.asarray(v, float) + (1 - beta2) * gt * gt
        v_hat = v_t / (1 - beta2 ** t)
        if kind == "extra_beta2":
            v_hat = beta2 * v_hat
        if nesterov_second_moment:
            v_hat = (beta2 * v_t / (1 - beta2 ** (t + 1))
                     + (1 - beta2) * gt * gt / (1 - beta2 ** t))
        u = m_hat / (np.sqrt(v_hat) + eps) + lam * x
        x_new, ratio, xn, un = O.layerwise_step(x, u, lr)
        return O.NLambResult(x_new, m_t, v_t, p_t, ratio, xn, un)
    return fn


@pytest.mark.parametrize("kind", ["schedule_as_power", "product_off_by_one",
                                  "no_gradient_term", "extra_beta2"])
def test_pins_reject_planted_mistake(kind):
    caught = any(not _matches(c, _run(c, _mutant(kind))) for c in _cases()
                 if not c["nesterov_second_moment"])
    rng = np.random.default_rng(9)
    w, g, m, v = _block(rng, 64)
    u, m_t, v_t, prod_t = _nadam_direction(w, g, m, v, 3, 0.9, 0.975, 0.999,
                                           1e-8, 0.004, 0.01)
    res = _mutant(kind)(w, g, m, v, t=3, lr=1e-3, mu_product=0.9)
    want = w - 1e-3 * np.linalg.norm(w) / np.linalg.norm(u) * u
    if not np.allclose(res.w, want, rtol=1e-12, atol=1e-18):
        caught = True
    assert caught, kind
