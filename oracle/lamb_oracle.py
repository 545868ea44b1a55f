"""Reference oracle for the layerwise-adaptive optimizer step (LAMB and LARS).

TEST INFRASTRUCTURE, NOT PRODUCT CODE.  Only the test suite, the smoke check
of the package entry point and the CPU-baseline leg of the benchmark may
import or run this module.  The CUDA library never calls it and shares no
code with it.

Everything here is plain NumPy in float64, one parameter block ("layer",
read as one parameter tensor) at a time, following the paper
"Large Batch Optimization for Deep Learning: Training BERT in 76 minutes"
(You et al., ICLR 2020):

* ``lamb_tensor``   -- Algorithm 2 (LAMB), steps in the algorithm's order;
                       ``lamb_direction`` is its element-wise part.
* ``nlamb_tensor``  -- Algorithms 3 and 4 of the appendix (N-LAMB, NN-LAMB:
                       Nesterov momentum in the first, or both, moments).
* ``lars_tensor``   -- Algorithm 1 (LARS); ``lars_momentum`` is its
                       element-wise part.
* ``layerwise_step``-- the general strategy of Section 3: a base update u is
                       normalised per block and rescaled by phi(||x||).
* ``phi``           -- the scaling function of Section 3,
                       phi(z) = min(max(z, gamma_l), gamma_u), or identity.
* ``block_norm``    -- the per-block l2 norm of Section 2 (Notation).
* ``bf16_rne``      -- round-to-nearest-even of float32 values to bfloat16
                       (the optional low-precision weight copy; the paper
                       is silent on it, see reading Q10 below).

Readings of the paper taken here (the paper is silent or ambiguous):

Q1  A block x^(i) is one parameter tensor.
Q2  Algorithm 2 writes the bias-corrected moments back into m_t, v_t.  The
    appendix ("LAMB with learning rate correction") calls this the original
    Adam correction, so the stored recurrences keep the *uncorrected* m_t,
    v_t and the correction is applied only where r_t is formed.
Q3  epsilon is added outside the square root: sqrt(v_hat) + eps.
Q4  Weight decay sits inside the normalised direction: u = r + lambda*x and
    the norm in the denominator is ||r + lambda*x||.
Q5  A per-tensor decay mask: lambda_k = lambda * mask_k.
Q6  If ||x|| == 0 or ||u|| == 0 the trust ratio is 1.
Q7  LARS takes an extra trust coefficient kappa: ratio = kappa*phi(||x||)/||m||
    (the paper's Algorithm 1 is kappa = 1).
Q8  Masked tensors still get the trust ratio; the mask removes decay only.
Q9  Bias correction uses beta**t in float64 with an integer t >= 1.
Q15 Non-finite inputs are not masked; NaN/Inf propagate.
Q16 Learning-rate schedule (Section 4: polynomial decay eta_t = eta_0 (1 -
    t/T) and linear warmup): eta_t = eta_0 t / T_w for t < T_w, else
    eta_0 max(0, 1 - t/T) -- the decay holds from step 0 and the warmup
    replaces it during the first T_w steps.
Q12 N-LAMB / NN-LAMB (appendix): the superscripted beta_1^t is the t-th term
    of a momentum schedule (the input line lists the schedule separately from
    the constant beta1 of the moment recurrence); it is Dozat's Nadam
    schedule, which the appendix cites and whose settings it uses:
    mu_t = beta1 * (1 - 0.5 * 0.96^(t * psi)).  The products prod_{i<=t} mu_i
    are carried from step to step as optimizer state.  N-LAMB keeps Adam's
    second moment ("the second moment of Adam was unchanged"), so its
    v_hat = v_t / (1 - beta2^t); the extra beta2 factor printed in Alg. 3 is
    read as a typo.  In NN-LAMB the second-moment schedule is constant
    (beta2), since the algorithm's inputs give none.

Q17 Gradient norms and the non-finite guard (not in the paper; the
    training-system checks that accompany a large-batch step): ||g_k|| per
    block, the global ||g|| = sqrt(sum_k ||g_k||^2) (the norm of the whole
    gradient viewed as one vector), and a decision "non-finite" when any
    element of any g_k is Inf or NaN.  A guarded step with that decision is
    not applied: x, m, v and t keep their values.
Q18 Decoupled weight decay (an ablation of Q4 the paper does not define;
    the AdamW-style decoupling applied to LAMB): the normalised direction is
    r alone, ratio = phi(||x||)/||r||, and x <- x - lr*ratio*r - lr*lam*x.

Input conventions: arrays may be float32 (or bfloat16 bit patterns given as
uint16 together with ``g_dtype="bf16"``); they are converted exactly to
float64 before any arithmetic.  Hyperparameters are Python floats.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np

__all__ = [
    "LambResult",
    "LarsResult",
    "phi",
    "block_norm",
    "to_f64",
    "bf16_bits_to_f64",
    "bf16_rne",
    "layerwise_step",
    "lamb_tensor",
    "lars_tensor",
    "lamb_tensor_scalar",
    "nadam_mu",
    "lr_schedule",
    "nlamb_tensor",
    "NLambResult",
    "lamb_step",
    "lars_step",
    "GradCheck",
    "grad_check",
]


# --------------------------------------------------------------------------
# Elementary pieces
# --------------------------------------------------------------------------

def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact value of bfloat16 bit patterns: the pattern is the top half of a
    float32, so widening by 16 zero bits gives the float32 of equal value."""
    b = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return b.view(np.float32).astype(np.float64)


def to_f64(x: np.ndarray, dtype: str = "f32") -> np.ndarray:
    """Exact widening of the stored input to float64."""
    if dtype == "bf16":
        return bf16_bits_to_f64(x)
    return np.asarray(x).astype(np.float64)


def bf16_rne(x32: np.ndarray) -> np.ndarray:
    """Round float32 values to bfloat16 (nearest, ties to even) and return the
    16-bit patterns.

    bfloat16 keeps the top 16 bits of the float32 encoding.  Rounding to
    nearest-even adds half a unit of the kept part (0x7FFF) plus the lowest
    kept bit, then truncates.  NaNs keep a quiet-NaN pattern.
    """
    f = np.ascontiguousarray(np.asarray(x32, dtype=np.float32))
    u = f.view(np.uint32).astype(np.uint64)
    lsb = (u >> np.uint64(16)) & np.uint64(1)
    rounded = ((u + np.uint64(0x7FFF) + lsb) >> np.uint64(16)).astype(np.uint16)
    nan = np.isnan(f)
    if nan.any():
        quiet = ((u >> np.uint64(16)) | np.uint64(0x0040)).astype(np.uint16)
        rounded = np.where(nan, quiet, rounded)
    return rounded


def phi(z: float, kind: str = "identity", gamma_l: float = 0.0,
        gamma_u: float = math.inf) -> float:
    """Section 3 scaling function: identity, or min(max(z, gamma_l), gamma_u).

    Comparisons are written so that a NaN input stays NaN (reading Q15)."""
    if kind == "identity":
        return z
    if kind != "clip":
        raise ValueError(f"unknown phi kind {kind!r}")
    if z < gamma_l:
        return gamma_l
    if z > gamma_u:
        return gamma_u
    return z


def block_norm(x: np.ndarray) -> float:
    """l2 norm of one block (Section 2, Notation): sqrt(sum_j x_j^2), summed
    in float64 by NumPy's pairwise reduction."""
    x = np.asarray(x, dtype=np.float64)
    return math.sqrt(float(np.sum(x * x)))


def layerwise_step(x: np.ndarray, u: np.ndarray, lr: float, *,
                   phi_kind: str = "identity", gamma_l: float = 0.0,
                   gamma_u: float = math.inf, trust_coef: float = 1.0):
    """General strategy of Section 3 for one block:
    x <- x - lr * kappa * phi(||x||) / ||u|| * u, ratio 1 if a norm is 0.

    Returns (x_new, ratio, ||x||, ||u||)."""
    x = np.asarray(x, dtype=np.float64)
    u = np.asarray(u, dtype=np.float64)
    xn = block_norm(x)
    un = block_norm(u)
    if xn == 0.0 or un == 0.0:
        ratio = 1.0
    else:
        ratio = trust_coef * phi(xn, phi_kind, gamma_l, gamma_u) / un
    return x - lr * ratio * u, ratio, xn, un


# --------------------------------------------------------------------------
# Algorithm 2 (LAMB) and Algorithm 1 (LARS), one block
# --------------------------------------------------------------------------

@dataclass
class LambResult:
    w: np.ndarray       # x_{t+1}
    m: np.ndarray       # uncorrected first moment m_t (reading Q2)
    v: np.ndarray       # uncorrected second moment v_t (reading Q2)
    ratio: float        # phi(||x||) / ||r + lambda x|| (1 on a zero norm)
    wnorm: float        # ||x_t||
    unorm: float        # ||r_t + lambda x_t||


@dataclass
class LarsResult:
    w: np.ndarray
    m: np.ndarray
    ratio: float
    wnorm: float
    unorm: float        # ||m_t||


def lamb_direction(w, g, m, v, *, t: int, beta1: float = 0.9,
                   beta2: float = 0.999, eps: float = 1e-6,
                   weight_decay: float = 0.01, decay: bool = True,
                   bias_correction: bool = True, g_dtype: str = "f32",
                   decoupled_decay: bool = False):
    """The element-wise part of Algorithm 2 for one block (or any slice of
    one): (m_t, v_t, u) in float64, u = r_t + lam x_t (r_t alone with
    decoupled decay, reading Q18).

      m_t = beta1 m_{t-1} + (1-beta1) g_t
      v_t = beta2 v_{t-1} + (1-beta2) g_t^2
      m_hat = m_t / (1 - beta1^t),  v_hat = v_t / (1 - beta2^t)
      r_t = m_hat / (sqrt(v_hat) + eps)
    """
    if t < 1:
        raise ValueError("step count t must be >= 1")
    x = to_f64(w)
    gt = to_f64(g, g_dtype)
    m_prev = to_f64(m)
    v_prev = to_f64(v)
    lam = weight_decay if decay else 0.0
    m_t = beta1 * m_prev + (1.0 - beta1) * gt
    v_t = beta2 * v_prev + (1.0 - beta2) * (gt * gt)
    if bias_correction:
        m_hat = m_t / (1.0 - beta1 ** t)
        v_hat = v_t / (1.0 - beta2 ** t)
    else:
        m_hat, v_hat = m_t, v_t
    r_t = m_hat / (np.sqrt(v_hat) + eps)
    return m_t, v_t, (r_t if decoupled_decay else r_t + lam * x)


def lamb_tensor(w, g, m, v, *, t: int, lr: float, beta1: float = 0.9,
                beta2: float = 0.999, eps: float = 1e-6,
                weight_decay: float = 0.01, decay: bool = True,
                phi_kind: str = "identity", gamma_l: float = 0.0,
                gamma_u: float = math.inf, bias_correction: bool = True,
                g_dtype: str = "f32",
                decoupled_decay: bool = False) -> LambResult:
    """One LAMB step (Algorithm 2) on one block, in float64.

    Order of operations follows the algorithm:
      m_t = beta1 m_{t-1} + (1-beta1) g_t
      v_t = beta2 v_{t-1} + (1-beta2) g_t^2
      m_hat = m_t / (1 - beta1^t),  v_hat = v_t / (1 - beta2^t)
      r_t = m_hat / (sqrt(v_hat) + eps)
      x_{t+1} = x_t - lr * phi(||x_t||) / ||r_t + lam x_t|| * (r_t + lam x_t)
    With decoupled_decay (reading Q18) the last line becomes
      x_{t+1} = x_t - lr * phi(||x_t||) / ||r_t|| * r_t - lr * lam * x_t
    """
    x = to_f64(w)
    lam = weight_decay if decay else 0.0
    m_t, v_t, u = lamb_direction(
        w, g, m, v, t=t, beta1=beta1, beta2=beta2, eps=eps,
        weight_decay=weight_decay, decay=decay,
        bias_correction=bias_correction, g_dtype=g_dtype,
        decoupled_decay=decoupled_decay)
    x_new, ratio, xn, un = layerwise_step(
        x, u, lr, phi_kind=phi_kind, gamma_l=gamma_l, gamma_u=gamma_u)
    if decoupled_decay:
        return LambResult(x_new - lr * lam * x, m_t, v_t, ratio, xn, un)
    return LambResult(x_new, m_t, v_t, ratio, xn, un)


def lars_tensor(w, g, m, *, lr: float, beta1: float = 0.9,
                weight_decay: float = 0.0, decay: bool = True,
                trust_coef: float = 1.0, phi_kind: str = "identity",
                gamma_l: float = 0.0, gamma_u: float = math.inf,
                g_dtype: str = "f32") -> LarsResult:
    """One LARS step (Algorithm 1) on one block, in float64.

      m_t = beta1 m_{t-1} + (1-beta1) (g_t + lam x_t)
      x_{t+1} = x_t - lr * kappa * phi(||x_t||) / ||m_t|| * m_t
    """
    x = to_f64(w)
    m_t = lars_momentum(w, g, m, beta1=beta1, weight_decay=weight_decay,
                        decay=decay, g_dtype=g_dtype)
    x_new, ratio, xn, un = layerwise_step(
        x, m_t, lr, phi_kind=phi_kind, gamma_l=gamma_l, gamma_u=gamma_u,
        trust_coef=trust_coef)
    return LarsResult(x_new, m_t, ratio, xn, un)


def lars_momentum(w, g, m, *, beta1: float = 0.9, weight_decay: float = 0.0,
                  decay: bool = True, g_dtype: str = "f32") -> np.ndarray:
    """The element-wise part of Algorithm 1 for one block (or any slice of
    one): m_t = beta1 m_{t-1} + (1-beta1) (g_t + lam x_t), float64."""
    x = to_f64(w)
    gt = to_f64(g, g_dtype)
    m_prev = to_f64(m)
    lam = weight_decay if decay else 0.0
    return beta1 * m_prev + (1.0 - beta1) * (gt + lam * x)


def lr_schedule(t: int, eta0: float, warmup: int, total: int) -> float:
    """Section 4 learning rate at step t (reading Q16)."""
    if warmup > 0 and t < warmup:
        return eta0 * t / warmup
    return eta0 * max(0.0, 1.0 - t / total)


def nadam_mu(t: int, beta1: float, psi: float) -> float:
    """Momentum schedule term mu_t = beta1 * (1 - 0.5 * 0.96^(t psi)) (Dozat's
    Nadam schedule; reading Q12 of the N-LAMB superscripts)."""
    return beta1 * (1.0 - 0.5 * 0.96 ** (t * psi))


@dataclass
class NLambResult:
    w: np.ndarray
    m: np.ndarray
    v: np.ndarray
    mu_product: float   # prod_{i <= t} mu_i, carried to the next step
    ratio: float
    wnorm: float
    unorm: float


def nlamb_tensor(w, g, m, v, *, t: int, lr: float, mu_product: float,
                 beta1: float = 0.975, beta2: float = 0.999, eps: float = 1e-8,
                 psi: float = 0.004, weight_decay: float = 0.01,
                 decay: bool = True, nesterov_second_moment: bool = False,
                 phi_kind: str = "identity", gamma_l: float = 0.0,
                 gamma_u: float = math.inf, g_dtype: str = "f32",
                 decoupled_decay: bool = False) -> NLambResult:
    """One N-LAMB (Algorithm 3) or, with nesterov_second_moment, NN-LAMB
    (Algorithm 4) step on one block, in float64.

    mu_product is prod_{i < t} mu_i from the previous steps (1 at t = 1).
      m_t   = beta1 m + (1-beta1) g
      m_hat = mu_{t+1} m_t / (1 - prod_{i<=t+1} mu_i)
              + (1 - mu_t) g / (1 - prod_{i<=t} mu_i)
      v_t   = beta2 v + (1-beta2) g^2
      v_hat = v_t / (1 - beta2^t)                                (N-LAMB)
            = beta2 v_t / (1 - beta2^(t+1)) + (1-beta2) g^2 / (1 - beta2^t)
                                                                 (NN-LAMB)
      r = m_hat / (sqrt(v_hat) + eps); then the layerwise step on r + lambda x
      (with decoupled_decay, reading Q18: on r, then x -= lr * lambda * x).
    """
    if t < 1:
        raise ValueError("step count t must be >= 1")
    x = to_f64(w)
    gt = to_f64(g, g_dtype)
    m_prev = to_f64(m)
    v_prev = to_f64(v)
    lam = weight_decay if decay else 0.0
    mu_t = nadam_mu(t, beta1, psi)
    mu_next = nadam_mu(t + 1, beta1, psi)
    prod_t = mu_product * mu_t
    prod_next = prod_t * mu_next
    m_t = beta1 * m_prev + (1.0 - beta1) * gt
    m_hat = mu_next * m_t / (1.0 - prod_next) + (1.0 - mu_t) * gt / (1.0 - prod_t)
    v_t = beta2 * v_prev + (1.0 - beta2) * (gt * gt)
    if nesterov_second_moment:
        v_hat = (beta2 * v_t / (1.0 - beta2 ** (t + 1))
                 + (1.0 - beta2) * (gt * gt) / (1.0 - beta2 ** t))
    else:
        v_hat = v_t / (1.0 - beta2 ** t)
    r_t = m_hat / (np.sqrt(v_hat) + eps)
    if decoupled_decay:
        x_new, ratio, xn, un = layerwise_step(
            x, r_t, lr, phi_kind=phi_kind, gamma_l=gamma_l, gamma_u=gamma_u)
        return NLambResult(x_new - lr * lam * x, m_t, v_t, prod_t, ratio, xn,
                           un)
    u = r_t + lam * x
    x_new, ratio, xn, un = layerwise_step(
        x, u, lr, phi_kind=phi_kind, gamma_l=gamma_l, gamma_u=gamma_u)
    return NLambResult(x_new, m_t, v_t, prod_t, ratio, xn, un)


def lamb_tensor_scalar(w, g, m, v, *, t, lr, beta1=0.9, beta2=0.999, eps=1e-6,
                       weight_decay=0.01, decay=True, phi_kind="identity",
                       gamma_l=0.0, gamma_u=math.inf, bias_correction=True):
    """Algorithm 2 again, one coordinate at a time with Python floats and
    ``math.fsum``.  Only for tiny blocks: it exists so the vectorised path can
    be checked against a loop that shares none of its array code."""
    n = len(w)
    lam = weight_decay if decay else 0.0
    c1 = 1.0 - beta1 ** t if bias_correction else 1.0
    c2 = 1.0 - beta2 ** t if bias_correction else 1.0
    m_out, v_out, u = [0.0] * n, [0.0] * n, [0.0] * n
    for j in range(n):
        gj = float(g[j])
        m_out[j] = beta1 * float(m[j]) + (1.0 - beta1) * gj
        v_out[j] = beta2 * float(v[j]) + (1.0 - beta2) * gj * gj
        rj = (m_out[j] / c1) / (math.sqrt(v_out[j] / c2) + eps)
        u[j] = rj + lam * float(w[j])
    wn = math.sqrt(math.fsum(float(x) * float(x) for x in w))
    un = math.sqrt(math.fsum(x * x for x in u))
    if wn == 0.0 or un == 0.0:
        ratio = 1.0
    else:
        ratio = phi(wn, phi_kind, gamma_l, gamma_u) / un
    w_out = [float(w[j]) - lr * ratio * u[j] for j in range(n)]
    return w_out, m_out, v_out, ratio


# --------------------------------------------------------------------------
# Whole-model steps: every block independently (Section 3: layerwise)
# --------------------------------------------------------------------------

def lamb_step(ws, gs, ms, vs, decay_mask, *, t, lr, g_dtype="f32", **hyper):
    """LAMB over a list of blocks; returns a list of LambResult."""
    return [lamb_tensor(w, g, m, v, t=t, lr=lr, decay=bool(d),
                        g_dtype=g_dtype, **hyper)
            for w, g, m, v, d in zip(ws, gs, ms, vs, decay_mask)]


def lars_step(ws, gs, ms, decay_mask, *, lr, g_dtype="f32", **hyper):
    """LARS over a list of blocks; returns a list of LarsResult."""
    return [lars_tensor(w, g, m, lr=lr, decay=bool(d), g_dtype=g_dtype,
                        **hyper)
            for w, g, m, d in zip(ws, gs, ms, decay_mask)]


# --------------------------------------------------------------------------
# Gradient norms and the non-finite guard (reading Q17)
# --------------------------------------------------------------------------

@dataclass
class GradCheck:
    norms: list         # ||g_k|| per block
    norm: float         # sqrt(sum_k ||g_k||^2)
    nonfinite: bool     # some element of some g_k is Inf or NaN


def grad_check(gs, g_dtype: str = "f32") -> GradCheck:
    """Per-block l2 norms of the gradient (the norm of Section 2's notation,
    one block at a time), the l2 norm of the whole gradient, and whether any
    element is Inf or NaN.  Each square of an fp32 or bf16 value is exact in
    float64; the per-block sums use NumPy's pairwise reduction and the sum
    over blocks is exactly rounded (math.fsum).  A non-finite element makes
    its block's norm Inf or NaN, as the arithmetic gives."""
    sq = []
    bad = False
    for g in gs:
        x = to_f64(g, g_dtype)
        if not np.all(np.isfinite(x)):
            bad = True
        sq.append(float(np.sum(x * x)))
    total = math.fsum(sq) if all(math.isfinite(s) for s in sq) else sum(sq)
    return GradCheck([math.sqrt(s) for s in sq], math.sqrt(total), bad)
