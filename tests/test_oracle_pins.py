"""Pins for the fp64 oracle: it is checked here against things other than
itself -- hand-derived exact cases, closed forms and invariants stated by the
paper, textbook special cases computed by a library (torch's AdamW and SGD
with momentum, torch's bfloat16 cast), and brute-force loops on tiny inputs.
A final group plants mistakes into copies of the oracle and shows that the
pins reject each of them.
"""
import json
import math
import os

import numpy as np
import pytest
import sympy

from oracle import lamb_oracle as O

HERE = os.path.dirname(os.path.abspath(__file__))
GOLDEN = os.path.join(HERE, "golden", "hand_cases.json")


def _ev(expr: str) -> float:
    return float(sympy.N(sympy.sympify(expr), 40))


def _load_cases():
    with open(GOLDEN) as f:
        return json.load(f)["cases"]


def _run_case(case, lamb_fn=None, lars_fn=None):
    lamb_fn = lamb_fn or O.lamb_tensor
    lars_fn = lars_fn or O.lars_tensor
    h = case["hyper"]
    arr = lambda key: np.array([_ev(s) for s in case[key]], dtype=np.float64)
    common = dict(lr=_ev(h["lr"]), beta1=_ev(h["beta1"]),
                  weight_decay=_ev(h["weight_decay"]), decay=h["decay"],
                  phi_kind=h["phi"], gamma_l=_ev(h.get("gamma_l", "0")),
                  gamma_u=_ev(h.get("gamma_u", "oo")))
    if case["algorithm"] == "lamb":
        if h.get("decoupled_decay"):
            common["decoupled_decay"] = True
        return lamb_fn(arr("w"), arr("g"), arr("m"), arr("v"), t=h["t"],
                       beta2=_ev(h["beta2"]), eps=_ev(h["eps"]),
                       bias_correction=h.get("bias_correction", True),
                       **common)
    return lars_fn(arr("w"), arr("g"), arr("m"),
                   trust_coef=_ev(h["trust_coef"]), **common)


def _case_matches(case, res, rtol=1e-12, atol=1e-15):
    exp = case["expected"]
    ok = True
    for key in ("w", "m", "v"):
        if key in exp:
            want = np.array([_ev(s) for s in exp[key]])
            ok &= np.allclose(getattr(res, key), want, rtol=rtol, atol=atol)
    for key in ("ratio", "wnorm", "unorm"):
        ok &= math.isclose(getattr(res, key), _ev(exp[key]), rel_tol=rtol,
                           abs_tol=atol)
    return bool(ok)


# ---------------------------------------------------------------------------
# P1: hand-derived exact cases (Algorithm 1, Algorithm 2)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("case", _load_cases(), ids=lambda c: c["name"])
def test_hand_case(case):
    res = _run_case(case)
    exp = case["expected"]
    for key in ("w", "m", "v"):
        if key in exp:
            want = np.array([_ev(s) for s in exp[key]])
            np.testing.assert_allclose(getattr(res, key), want, rtol=1e-12,
                                       atol=1e-15, err_msg=key)
    for key in ("ratio", "wnorm", "unorm"):
        assert math.isclose(getattr(res, key), _ev(exp[key]), rel_tol=1e-12,
                            abs_tol=1e-15), key


# ---------------------------------------------------------------------------
# Helpers: random blocks
# ---------------------------------------------------------------------------

def _rand_block(rng, n, gscale=1e-3, warm=True):
    w = rng.normal(0, 0.02, n)
    g = rng.normal(0, gscale, n)
    if warm:
        m = rng.normal(0, 0.3 * gscale, n)
        v = (gscale ** 2) * rng.uniform(0.0005, 0.003, n)
    else:
        m = np.zeros(n)
        v = np.zeros(n)
    return w, g, m, v


# ---------------------------------------------------------------------------
# P2: ||x' - x|| = lr * phi(||x||) when both norms are nonzero (Section 3;
# the proofs of Theorems 2 and 3 use exactly this normalised step)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("phi_kind,gl,gu", [("identity", 0.0, math.inf),
                                            ("clip", 0.0, 10.0),
                                            ("clip", 0.5, 0.6),
                                            ("clip", 0.0, 1e-3)])
@pytest.mark.parametrize("n", [1, 7, 1000, 65537])
def test_step_norm_closed_form(phi_kind, gl, gu, n):
    rng = np.random.default_rng(n)
    w, g, m, v = _rand_block(rng, n)
    lr = 2e-3
    res = O.lamb_tensor(w, g, m, v, t=4, lr=lr, phi_kind=phi_kind,
                        gamma_l=gl, gamma_u=gu)
    step = math.sqrt(float(np.sum((res.w - w) ** 2)))
    target = lr * min(max(np.linalg.norm(w), gl), gu)
    assert math.isclose(step, target, rel_tol=1e-9)
    lres = O.lars_tensor(w, g, m, lr=lr, weight_decay=1e-4, trust_coef=1.0,
                         phi_kind=phi_kind, gamma_l=gl, gamma_u=gu)
    step = math.sqrt(float(np.sum((lres.w - w) ** 2)))
    assert math.isclose(step, target, rel_tol=1e-9)


def test_step_norm_closed_form_trust_coef():
    rng = np.random.default_rng(3)
    w, g, m, _ = _rand_block(rng, 333)
    res = O.lars_tensor(w, g, m, lr=0.1, weight_decay=1e-4, trust_coef=1e-3)
    step = np.linalg.norm(res.w - w)
    assert math.isclose(step, 0.1 * 1e-3 * np.linalg.norm(w), rel_tol=1e-9)


# ---------------------------------------------------------------------------
# P3: beta1 = beta2 = 0 reduces LAMB to sign-SGD scaled by sqrt(d)
# (Section 3, discussion under Algorithm 2)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("n", [1, 5, 4096])
def test_sign_sgd_reduction(n):
    rng = np.random.default_rng(10 + n)
    w, g, _, _ = _rand_block(rng, n, warm=False)
    g[1::7] = 0.0                                # some exact zeros
    m = rng.normal(0, 1, n)                      # ignored when beta = 0
    v = rng.uniform(0, 1, n)
    lr = 1e-2
    res = O.lamb_tensor(w, g, m, v, t=3, lr=lr, beta1=0.0, beta2=0.0,
                        eps=0.0 + 1e-300, weight_decay=0.0)
    nz = np.count_nonzero(g)
    # r_j = g_j / (|g_j| + eps) = sign(g_j) to within eps/|g_j|
    r = res.m / (np.sqrt(res.v) + 1e-300)
    np.testing.assert_allclose(r, np.sign(g), rtol=1e-12, atol=0)
    assert math.isclose(res.unorm, math.sqrt(nz), rel_tol=1e-12)
    expect = w - lr * np.linalg.norm(w) / math.sqrt(nz) * np.sign(g)
    np.testing.assert_allclose(res.w, expect, rtol=1e-12, atol=1e-18)


def test_sign_sgd_with_eps():
    rng = np.random.default_rng(11)
    w, g, _, _ = _rand_block(rng, 1000, warm=False)
    eps = 1e-6
    res = O.lamb_tensor(w, g, np.zeros(1000), np.zeros(1000), t=1, lr=1e-3,
                        beta1=0.0, beta2=0.0, eps=eps, weight_decay=0.0)
    # |r_j| = |g_j|/(|g_j|+eps) = 1 - O(eps/|g_j|)
    dev = abs(res.unorm - math.sqrt(1000)) / math.sqrt(1000)
    assert dev <= np.max(eps / np.abs(g))
    assert dev > 0


# ---------------------------------------------------------------------------
# P4: with u = g the strategy is the LARS-style normalised step (Section 3
# general strategy with base SGD; proof of Theorem 2).  LAMB produces u
# proportional to g when beta1 = 0 and sqrt(v_t) is the same for every
# coordinate, so LAMB, LARS(beta1=0, lambda=0, kappa=1) and the general
# strategy must coincide.
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("phi_kind,gu", [("identity", math.inf), ("clip", 0.3)])
def test_lamb_reduces_to_normalised_sgd(phi_kind, gu):
    rng = np.random.default_rng(21)
    n = 513
    w, g, _, _ = _rand_block(rng, n)
    beta2 = 0.5
    C = 4.0 * float(np.max(g * g))
    v_prev = (C - (1 - beta2) * g * g) / beta2   # makes v_t == C
    lr = 3e-3
    lamb = O.lamb_tensor(w, g, np.zeros(n), v_prev, t=9, lr=lr, beta1=0.0,
                         beta2=beta2, eps=0.0, weight_decay=0.0,
                         bias_correction=False, phi_kind=phi_kind, gamma_u=gu)
    np.testing.assert_allclose(lamb.v, C, rtol=1e-14)
    lars = O.lars_tensor(w, g, np.zeros(n), lr=lr, beta1=0.0,
                         weight_decay=0.0, trust_coef=1.0, phi_kind=phi_kind,
                         gamma_u=gu)
    np.testing.assert_allclose(lamb.w, lars.w, rtol=1e-13, atol=1e-19)
    # and the plain SGD-based strategy x - lr*phi(||x||)/||g|| * g
    ph = min(np.linalg.norm(w), gu)
    want = w - lr * ph / np.linalg.norm(g) * g
    np.testing.assert_allclose(lars.w, want, rtol=1e-13, atol=1e-19)


# ---------------------------------------------------------------------------
# P5: with beta1 = 0 (no correction) ||r|| <= sqrt(d/(1-beta2)) for every
# block and every step (proof of Theorem 3)
# ---------------------------------------------------------------------------

def test_ratio_norm_bound_along_trajectory():
    rng = np.random.default_rng(5)
    sizes = [1, 3, 100, 4097]
    beta2 = 0.99
    state = [(rng.normal(0, 0.02, d), np.zeros(d), np.zeros(d)) for d in sizes]
    for t in range(1, 21):
        new = []
        for (w, m, v), d in zip(state, sizes):
            g = rng.normal(0, 10 ** rng.uniform(-5, 0), d)
            res = O.lamb_tensor(w, g, m, v, t=t, lr=1e-2, beta1=0.0,
                                beta2=beta2, eps=0.0 + 1e-30,
                                weight_decay=0.0, bias_correction=False)
            assert res.unorm <= math.sqrt(d / (1 - beta2)) * (1 + 1e-12)
            new.append((res.w, res.m, res.v))
        state = new


# ---------------------------------------------------------------------------
# P6: zero-norm rules on blocks of several sizes (reading Q6)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("n", [1, 2, 1000])
def test_zero_norm_rules(n):
    rng = np.random.default_rng(n)
    w, g, m, v = _rand_block(rng, n, warm=False)
    z = np.zeros(n)
    r = O.lamb_tensor(z, g, m, v, t=1, lr=1e-2)          # w == 0
    assert r.ratio == 1.0 and r.wnorm == 0.0
    u = r.m / (1 - 0.9) / (np.sqrt(r.v / (1 - 0.999)) + 1e-6)
    np.testing.assert_allclose(r.w, -1e-2 * u, rtol=1e-13)
    r = O.lamb_tensor(w, z, z, z, t=1, lr=1e-2, decay=False)   # r == 0
    assert r.ratio == 1.0 and r.unorm == 0.0
    np.testing.assert_array_equal(r.w, w)
    r = O.lamb_tensor(w, z, z, z, t=1, lr=1e-2, weight_decay=0.01)
    assert math.isclose(np.linalg.norm(r.w - w), 1e-2 * np.linalg.norm(w),
                        rel_tol=1e-12)
    r = O.lamb_tensor(z, g, m, v, t=1, lr=1e-2, phi_kind="clip",
                      gamma_l=0.5, gamma_u=2.0)               # clip, w == 0
    assert r.ratio == 1.0
    lr_ = O.lars_tensor(z, g, z, lr=1e-2, weight_decay=0.1, trust_coef=1e-3)
    assert lr_.ratio == 1.0
    lr_ = O.lars_tensor(w, z, z, lr=1e-2, weight_decay=0.0)
    assert lr_.ratio == 1.0
    np.testing.assert_array_equal(lr_.w, w)


# ---------------------------------------------------------------------------
# P7: bias correction becomes the identity at large t (appendix "LAMB with
# learning rate correction": it acts like warmup only early on)
# ---------------------------------------------------------------------------

def test_bias_correction_vanishes_at_large_t():
    rng = np.random.default_rng(7)
    w, g, m, v = _rand_block(rng, 2000)
    a = O.lamb_tensor(w, g, m, v, t=100000, lr=1e-3, bias_correction=True)
    b = O.lamb_tensor(w, g, m, v, t=100000, lr=1e-3, bias_correction=False)
    np.testing.assert_allclose(a.w, b.w, rtol=1e-14, atol=0)
    c = O.lamb_tensor(w, g, m, v, t=1, lr=1e-3, bias_correction=True)
    assert not np.allclose(c.w, b.w, rtol=1e-9, atol=0)


# ---------------------------------------------------------------------------
# P8: the Adam ratio is scale free for eps = 0, so scaling every gradient of
# a trajectory by c > 0 leaves the weights unchanged (Algorithm 2, ratio
# line).  A power of two scales exactly, so the trajectories are bitwise
# equal; c = 3 holds to round-off.
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("c,exact", [(8.0, True), (3.0, False)])
def test_gradient_scale_invariance(c, exact):
    rng = np.random.default_rng(8)
    n = 777
    w0 = rng.normal(0, 0.02, n)
    gs = [rng.normal(0, 1e-3, n) for _ in range(5)]
    def run(scale):
        w, m, v = w0.copy(), np.zeros(n), np.zeros(n)
        for t, g in enumerate(gs, start=1):
            r = O.lamb_tensor(w, scale * g, m, v, t=t, lr=1e-3, eps=0.0,
                              weight_decay=0.01)
            w, m, v = r.w, r.m, r.v
        return w
    a, b = run(1.0), run(c)
    if exact:
        np.testing.assert_array_equal(a, b)
    else:
        np.testing.assert_allclose(a, b, rtol=1e-13)


# ---------------------------------------------------------------------------
# P9: vectorised oracle == scalar Python loop with math.fsum
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("seed", range(6))
def test_vectorised_equals_scalar_loop(seed):
    rng = np.random.default_rng(100 + seed)
    n = int(rng.integers(1, 40))
    w, g, m, v = _rand_block(rng, n)
    kw = dict(t=int(rng.integers(1, 50)), lr=1e-3, weight_decay=0.01,
              decay=bool(seed % 2), phi_kind="clip" if seed % 3 else "identity",
              gamma_l=0.0, gamma_u=0.05, bias_correction=seed != 4)
    res = O.lamb_tensor(w, g, m, v, **kw)
    w2, m2, v2, ratio2 = O.lamb_tensor_scalar(w, g, m, v, **kw)
    np.testing.assert_allclose(res.w, w2, rtol=1e-14, atol=1e-20)
    np.testing.assert_allclose(res.m, m2, rtol=1e-15, atol=0)
    np.testing.assert_allclose(res.v, v2, rtol=1e-15, atol=0)
    assert math.isclose(res.ratio, ratio2, rel_tol=1e-13)


# ---------------------------------------------------------------------------
# Library pins.  LAMB's direction u = r + lambda*x is exactly the per-element
# update of AdamW (Adam with decoupled weight decay) at learning rate 1, and
# LARS's m_t is heavy-ball momentum with dampening beta1 and L2 decay.
# torch's CPU optimizers in float64 compute those textbook updates.
# ---------------------------------------------------------------------------

torch = pytest.importorskip("torch")


def _close_to_operands(got, want, scale, rel=1e-14):
    err = np.abs(got - want)
    assert np.all(err <= rel * np.maximum(scale, np.abs(want))), \
        float(np.max(err / np.maximum(scale, np.abs(want))))


def _adamw_direction(w, g, m, v, t, beta1, beta2, eps, wd):
    p = torch.tensor(w, dtype=torch.float64, requires_grad=True)
    opt = torch.optim.AdamW([p], lr=1.0, betas=(beta1, beta2), eps=eps,
                            weight_decay=wd)
    opt.state[p] = {"step": torch.tensor(float(t - 1), dtype=torch.float64),
                    "exp_avg": torch.tensor(m, dtype=torch.float64),
                    "exp_avg_sq": torch.tensor(v, dtype=torch.float64)}
    p.grad = torch.tensor(g, dtype=torch.float64)
    opt.step()
    st = opt.state[p]
    u = w - p.detach().numpy()
    return u, st["exp_avg"].numpy(), st["exp_avg_sq"].numpy()


@pytest.mark.parametrize("decay", [True, False])
@pytest.mark.parametrize("t", [1, 2, 1000])
def test_lamb_direction_is_adamw_update(decay, t):
    rng = np.random.default_rng(t + 2 * decay)
    n = 301
    w, g, m, v = _rand_block(rng, n)
    if t == 1:
        m[:] = 0
        v[:] = 0
    wd = 0.01
    u, m_t, v_t = _adamw_direction(w, g, m, v, t, 0.9, 0.999, 1e-6,
                                   wd if decay else 0.0)
    lr = 2e-3
    res = O.lamb_tensor(w, g, m, v, t=t, lr=lr, weight_decay=wd, decay=decay,
                        phi_kind="clip", gamma_l=0.0, gamma_u=10.0)
    # torch forms m_t as a lerp; compare relative to the operands' size
    _close_to_operands(res.m, m_t, 0.9 * np.abs(m) + 0.1 * np.abs(g))
    np.testing.assert_allclose(res.v, v_t, rtol=1e-14, atol=0)
    assert math.isclose(res.unorm, np.linalg.norm(u), rel_tol=1e-10)
    want = w - lr * min(np.linalg.norm(w), 10.0) / np.linalg.norm(u) * u
    np.testing.assert_allclose(res.w, want, rtol=1e-12, atol=1e-18)


@pytest.mark.parametrize("wd", [0.0, 1e-4, 0.05])
def test_lars_momentum_is_sgd_momentum(wd):
    rng = np.random.default_rng(int(wd * 1e5) + 1)
    n = 257
    w, g, m, _ = _rand_block(rng, n)
    p = torch.tensor(w, dtype=torch.float64, requires_grad=True)
    opt = torch.optim.SGD([p], lr=1.0, momentum=0.9, dampening=0.9,
                          weight_decay=wd)
    opt.state[p] = {"momentum_buffer": torch.tensor(m, dtype=torch.float64)}
    p.grad = torch.tensor(g, dtype=torch.float64)
    opt.step()
    buf = opt.state[p]["momentum_buffer"].numpy()
    res = O.lars_tensor(w, g, m, lr=0.5, beta1=0.9, weight_decay=wd,
                        trust_coef=1e-3)
    _close_to_operands(res.m, buf,
                       0.9 * np.abs(m) + 0.1 * (np.abs(g) + wd * np.abs(w)))
    want = w - 0.5 * 1e-3 * np.linalg.norm(w) / np.linalg.norm(buf) * buf
    np.testing.assert_allclose(res.w, want, rtol=1e-13, atol=1e-20)


def test_bf16_rne_matches_torch_cast():
    rng = np.random.default_rng(12)
    vals = np.concatenate([
        rng.normal(0, 1, 20000).astype(np.float32),
        rng.normal(0, 1e-3, 20000).astype(np.float32),
        (rng.normal(0, 1, 5000) * 1e-38).astype(np.float32),   # subnormals
        np.array([0.0, -0.0, 1.0, -1.0, np.inf, -np.inf, 3.4e38, -3.4e38,
                  1e-45, 65504.0], dtype=np.float32),
    ])
    # exact ties: low 16 bits == 0x8000, with even and odd kept parts
    hi = rng.integers(0, 0x7F7F, 2000, dtype=np.uint32) << np.uint32(16)
    ties = (hi | np.uint32(0x8000)).view(np.float32)
    vals = np.concatenate([vals, ties, -ties])
    ours = O.bf16_rne(vals)
    ref = torch.from_numpy(vals).to(torch.bfloat16).view(torch.int16).numpy()
    np.testing.assert_array_equal(ours, ref.view(np.uint16))
    nan = O.bf16_rne(np.array([np.nan], dtype=np.float32))
    assert (int(nan[0]) & 0x7F80) == 0x7F80 and (int(nan[0]) & 0x7F) != 0


def test_bf16_widening_matches_torch():
    rng = np.random.default_rng(13)
    bits = rng.integers(0, 2 ** 16, 50000, dtype=np.uint16)
    bits = bits[(bits & 0x7F80) != 0x7F80]       # drop inf/nan patterns
    ours = O.bf16_bits_to_f64(bits)
    ref = torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).double()
    np.testing.assert_array_equal(ours, ref.numpy())


def test_phi_nan_propagates():
    assert math.isnan(O.phi(float("nan"), "clip", 0.0, 10.0))
    assert O.phi(20.0, "clip", 0.0, 10.0) == 10.0
    assert O.phi(-1.0, "clip", 0.0, 10.0) == 0.0
    with pytest.raises(ValueError):
        O.phi(1.0, "l1")


def test_step_count_must_be_positive():
    with pytest.raises(ValueError):
        O.lamb_tensor(np.ones(2), np.ones(2), np.zeros(2), np.zeros(2), t=0,
                      lr=1e-3)


# ---------------------------------------------------------------------------
# Planted mistakes: each mutant is the oracle with one plausible error; at
# least one pin above must reject it.
# ---------------------------------------------------------------------------

def _mutant(kind):
    def lamb(w, g, m, v, *, t, lr, beta1=0.9, beta2=0.999, eps=1e-6,
             weight_decay=0.01, decay=True, phi_kind="identity", gamma_l=0.0,
             gamma_u=math.inf, bias_correction=True, g_dtype="f32"):
        x = O.to_f64(w); gt = O.to_f64(g, g_dtype)
        m0 = O.to_f64(m); v0 = O.to_f64(v)
        lam = weight_decay if decay else 0.0
        if kind == "decay_ignores_mask":
            lam = weight_decay
        m_t = beta1 * m0 + (1 - beta1) * gt
        if kind == "no_m_damping":
            m_t = beta1 * m0 + gt
        v_t = beta2 * v0 + (1 - beta2) * gt * gt
        if kind == "swapped_betas":
            m_t = beta2 * m0 + (1 - beta2) * gt
            v_t = beta1 * v0 + (1 - beta1) * gt * gt
        c1 = 1 - beta1 ** t if bias_correction else 1.0
        c2 = 1 - beta2 ** t if bias_correction else 1.0
        if kind == "t_off_by_one":
            c1 = 1 - beta1 ** (t + 1) if bias_correction else 1.0
            c2 = 1 - beta2 ** (t + 1) if bias_correction else 1.0
        m_h, v_h = m_t / c1, v_t / c2
        if kind == "eps_inside_sqrt":
            r = m_h / np.sqrt(v_h + eps)
        else:
            r = m_h / (np.sqrt(v_h) + eps)
        u = r + lam * x
        if kind == "decay_sign":
            u = r - lam * x
        if kind == "norm_of_r_only":
            xn, un = O.block_norm(x), O.block_norm(r)
            ratio = 1.0 if xn == 0 or un == 0 else O.phi(xn, phi_kind, gamma_l,
                                                         gamma_u) / un
            return O.LambResult(x - lr * ratio * u, m_t, v_t, ratio, xn, un)
        if kind == "store_corrected":
            m_t, v_t = m_h, v_h
        xn, un = O.block_norm(x), O.block_norm(u)
        if kind == "zero_rule_zero":
            ratio = 0.0 if xn == 0 or un == 0 else O.phi(
                xn, phi_kind, gamma_l, gamma_u) / un
        else:
            ratio = 1.0 if xn == 0 or un == 0 else O.phi(
                xn, phi_kind, gamma_l, gamma_u) / un
        return O.LambResult(x - lr * ratio * u, m_t, v_t, ratio, xn, un)
    return lamb


@pytest.mark.parametrize("kind", ["decay_ignores_mask", "no_m_damping",
                                  "swapped_betas", "t_off_by_one",
                                  "eps_inside_sqrt", "decay_sign",
                                  "norm_of_r_only", "store_corrected",
                                  "zero_rule_zero"])
def test_pins_reject_planted_mistake(kind):
    mutant = _mutant(kind)
    caught = False
    for case in _load_cases():
        if case["algorithm"] != "lamb" or case["hyper"].get("decoupled_decay"):
            continue
        if not _case_matches(case, _run_case(case, lamb_fn=mutant)):
            caught = True
    # library pin (AdamW) at t = 2 with decay on and off
    rng = np.random.default_rng(99)
    w, g, m, v = _rand_block(rng, 64)
    for decay in (True, False):
        u, m_t, v_t = _adamw_direction(w, g, m, v, 2, 0.9, 0.999, 1e-6,
                                       0.01 if decay else 0.0)
        res = mutant(w, g, m, v, t=2, lr=1e-3, decay=decay)
        want = w - 1e-3 * np.linalg.norm(w) / np.linalg.norm(u) * u
        if not (np.allclose(res.w, want, rtol=1e-12, atol=1e-18)
                and np.allclose(res.m, m_t, rtol=1e-14)
                and np.allclose(res.v, v_t, rtol=1e-14)):
            caught = True
    assert caught, f"planted mistake {kind!r} passed every pin"



def _lars_mutant(kind):
    """Algorithm 1 with one plausible error planted."""
    def lars(w, g, m, *, lr, beta1=0.9, weight_decay=0.0, decay=True,
             trust_coef=1.0, phi_kind="identity", gamma_l=0.0,
             gamma_u=math.inf, g_dtype="f32"):
        x = O.to_f64(w); gt = O.to_f64(g, g_dtype); m0 = O.to_f64(m)
        lam = weight_decay if (decay or kind == "decay_ignores_mask") else 0.0
        if kind == "no_m_damping":
            m_t = beta1 * m0 + gt + lam * x
        elif kind == "decay_outside_momentum":
            m_t = beta1 * m0 + (1 - beta1) * gt
        else:
            m_t = beta1 * m0 + (1 - beta1) * (gt + lam * x)
        u = m_t + lam * x if kind == "decay_outside_momentum" else m_t
        xn, un = O.block_norm(x), O.block_norm(u)
        if kind == "norm_of_g":
            un = O.block_norm(gt)
        kappa = 1.0 if kind == "no_trust_coef" else trust_coef
        if xn == 0 or un == 0:
            ratio = 0.0 if kind == "zero_rule_zero" else 1.0
        elif kind == "norms_swapped":
            ratio = kappa * O.phi(un, phi_kind, gamma_l, gamma_u) / xn
        else:
            ratio = kappa * O.phi(xn, phi_kind, gamma_l, gamma_u) / un
        sign = 1.0 if kind == "update_sign" else -1.0
        return O.LarsResult(x + sign * lr * ratio * u, m_t, ratio, xn, un)
    return lars


@pytest.mark.parametrize("kind", ["decay_ignores_mask", "no_m_damping",
                                  "decay_outside_momentum", "norm_of_g",
                                  "no_trust_coef", "zero_rule_zero",
                                  "norms_swapped", "update_sign"])
def test_pins_reject_planted_lars_mistake(kind):
    mutant = _lars_mutant(kind)
    caught = False
    for case in _load_cases():
        if case["algorithm"] != "lars":
            continue
        if not _case_matches(case, _run_case(case, lars_fn=mutant)):
            caught = True
    # library pin: torch SGD momentum with dampening beta1 and L2 decay, and
    # the step-norm closed form with the trust coefficient
    rng = np.random.default_rng(98)
    w, g, m, _ = _rand_block(rng, 96)
    for wd in (0.0, 0.05):
        p = torch.tensor(w, dtype=torch.float64, requires_grad=True)
        opt = torch.optim.SGD([p], lr=1.0, momentum=0.9, dampening=0.9,
                              weight_decay=wd)
        opt.state[p] = {"momentum_buffer": torch.tensor(m, dtype=torch.float64)}
        p.grad = torch.tensor(g, dtype=torch.float64)
        opt.step()
        buf = opt.state[p]["momentum_buffer"].numpy()
        res = mutant(w, g, m, lr=0.5, beta1=0.9, weight_decay=wd,
                     trust_coef=1e-3)
        want = w - 0.5 * 1e-3 * np.linalg.norm(w) / np.linalg.norm(buf) * buf
        if not (np.allclose(res.m, buf, rtol=1e-13, atol=1e-20)
                and np.allclose(res.w, want, rtol=1e-12, atol=1e-20)):
            caught = True
    res = mutant(w, g, m, lr=0.1, weight_decay=1e-4, trust_coef=1e-3)
    if not math.isclose(np.linalg.norm(res.w - w), 0.1 * 1e-3 * np.linalg.norm(w),
                        rel_tol=1e-9):
        caught = True
    assert caught, f"planted LARS mistake {kind!r} passed every pin"

def test_unmutated_oracle_passes_pin_harness():
    for case in _load_cases():
        assert _case_matches(case, _run_case(case)), case["name"]


# ---------------------------------------------------------------------------
# Section 4 learning-rate schedule (reading Q16)
# ---------------------------------------------------------------------------

def test_lr_schedule_closed_forms():
    eta0, tw, T = 5e-3, 100, 1000
    assert O.lr_schedule(50, eta0, tw, T) == pytest.approx(eta0 * 0.5, rel=1e-15)
    assert O.lr_schedule(1, eta0, tw, T) == pytest.approx(eta0 / 100, rel=1e-15)
    assert O.lr_schedule(100, eta0, tw, T) == pytest.approx(eta0 * 0.9, rel=1e-15)
    assert O.lr_schedule(1000, eta0, tw, T) == 0.0
    assert O.lr_schedule(5000, eta0, tw, T) == 0.0
    assert O.lr_schedule(10, eta0, 0, T) == pytest.approx(eta0 * 0.99, rel=1e-15)


def test_lr_schedule_decay_is_torch_polynomial_lr():
    """After warmup the decay is torch's PolynomialLR with power 1."""
    p = torch.zeros(1, requires_grad=True)
    opt = torch.optim.SGD([p], lr=2e-3)
    sch = torch.optim.lr_scheduler.PolynomialLR(opt, total_iters=500, power=1.0)
    for t in range(0, 600):
        if t >= 1:
            opt.step()
            sch.step()
        assert O.lr_schedule(t, 2e-3, 0, 500) == pytest.approx(
            opt.param_groups[0]["lr"], rel=1e-12, abs=1e-18), t
