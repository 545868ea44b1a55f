"""GPU parity of the optional step variants against the fp64 oracle:

* the gradient check (per-tensor and global ||g||, Inf/NaN decision) fused
  into pass 1 (oracle reading Q17);
* the skip-on-non-finite mode, in which a step whose gradients hold an Inf
  or NaN writes nothing, and a finite step is bit-identical to the plain one;
* decoupled weight decay (oracle reading Q18), for LAMB and N-LAMB.
"""
import math

import numpy as np
import pytest
import torch

from gpu_util import (TOL_RATIO, TOL_STEP, GpuLayout, c_hyper, check_copy,
                      compare_lamb, compare_lars, compare_nlamb, f32,
                      hyper_kwargs, oracle_map, ratio_ok)
from oracle import lamb_oracle as O
from paper_1904_00962_gb300 import binding as B
from paper_1904_00962_gb300 import build as build_mod
from paper_1904_00962_gb300 import workloads as W

pytestmark = pytest.mark.gpu

SIZES = [0, 1, 3, 5, 1023, 1024, 16383, 16384, 16385, 65539, 0, 3000, 100003]


@pytest.fixture(scope="module", autouse=True)
def _lib(gpu):
    build_mod.build()
    B.load()
    yield
    torch.cuda.empty_cache()


def _layout(grad_dtype="f32", copy_dtype=None):
    n = len(SIZES)
    return W.Layout(name="variants", names=[f"t{i}" for i in range(n)],
                    shapes=[(s,) for s in SIZES],
                    decay=[(i + 1) % 2 for i in range(n)],
                    init=[("normal", 0.02)] * n,
                    grad_sigma=[10 ** (-2 - (i % 4)) for i in range(n)],
                    grad_dtype=grad_dtype, copy_dtype=copy_dtype,
                    zero_w={3}, zero_g={4},
                    hyper=W.Hyper(lr=2e-3, phi="clip", gamma_l=0.0,
                                  gamma_u=10.0))


def _hyper(h, lars=False, **flags):
    return B.make_hyper(beta1=h.beta1, beta2=h.beta2, eps=h.eps,
                        weight_decay=h.weight_decay, phi=h.phi,
                        gamma_l=h.gamma_l, gamma_u=h.gamma_u,
                        trust_coef=h.trust_coef,
                        bias_correction=(h.bias_correction and not lars),
                        **flags)


def _state(G):
    torch.cuda.synchronize()
    out = [G.st.w.clone(), G.st.m.clone()]
    if G.st.v is not None:
        out.append(G.st.v.clone())
    if G.st.copy is not None:
        out.append(G.st.copy.clone())
    return out


def _bitwise_equal(a, b):
    return all(torch.equal(x.view(torch.int8), y.view(torch.int8))
               for x, y in zip(a, b))


def _grad_norms(G):
    gn, gg, nf = G.plan.grad_norms()
    torch.cuda.synchronize()
    return gn.cpu().numpy(), float(gg.item()), int(nf.item())


def _prepared(L, step=2, **kw):
    G = GpuLayout(L, **kw)
    G.load_weights()
    G.load_warm_state()
    G.load_grads(step)
    return G


# ---------------------------------------------------------------------------
# Gradient check
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("grad_dtype,copy_dtype", [("f32", None),
                                                    ("bf16", "bf16")])
@pytest.mark.parametrize("algo", [1, 3], ids=["two_pass_plan",
                                              "on_chip_plan"])
@pytest.mark.parametrize("lars", [False, True], ids=["lamb", "lars"])
def test_grad_norms_match_oracle_and_leave_the_step_unchanged(
        grad_dtype, copy_dtype, algo, lars):
    L = _layout(grad_dtype, copy_dtype)
    h = L.hyper if not lars else W.Hyper(lr=0.5, trust_coef=1e-3,
                                         weight_decay=1e-4,
                                         bias_correction=False)
    lr = f32(h.lr)
    plain = _prepared(L, with_v=not lars)
    plain.step(2, lr, _hyper(h, lars), lars=lars)
    want_state = _state(plain)
    want_ratio = plain.results()[0]
    plain.close()

    G = _prepared(L, with_v=not lars, algorithm=algo)
    G.step(2, lr, _hyper(h, lars, grad_norm=True), lars=lars)
    ratio = G.results()[0]
    assert _bitwise_equal(_state(G), want_state)
    assert np.array_equal(ratio, want_ratio)
    gn, gg, nf = _grad_norms(G)
    ref = O.grad_check([L.grad(k, 2) for k in range(L.n_tensors)],
                       g_dtype=grad_dtype)
    assert nf == 0 and G.plan.query() == 0
    for k in range(L.n_tensors):
        assert ratio_ok(gn[k], ref.norms[k]), (k, gn[k], ref.norms[k])
    assert ratio_ok(gg, ref.norm), (gg, ref.norm)
    assert gn[0] == 0.0 and gn[4] == 0.0       # empty tensor, zero gradient
    G.close()


def test_grad_norms_bert_large_full_size():
    """BERT-large (bf16 g, bf16 copy): per-tensor and global ||g|| against
    the oracle at full size, in the launch configuration the benchmark
    times, and the step is bit-identical to the plain one."""
    L = W.bert_large_layout()
    h = L.hyper
    t = 1000
    lr = f32(h.lr)
    G = _prepared(L, step=t)
    before = _state(G)
    G.step(t, lr, _hyper(h))
    want = _state(G)
    for name, x in zip(("w", "m", "v", "copy"), before):
        getattr(G.st, name).copy_(x)
    G.step(t, lr, _hyper(h, grad_norm=True))
    assert _bitwise_equal(_state(G), want)
    del before, want
    gn, gg, nf = _grad_norms(G)
    assert nf == 0 and G.plan.query() == 0
    refs = oracle_map(lambda k: O.grad_check([L.grad(k, t)], "bf16").norms[0],
                      range(L.n_tensors))
    for k in range(L.n_tensors):
        assert ratio_ok(gn[k], refs[k]), (k, gn[k], refs[k])
    assert ratio_ok(gg, math.sqrt(math.fsum(r * r for r in refs)))
    G.close()


def test_grad_norm_flags_nonfinite_without_skipping():
    L = _layout()
    G = _prepared(L)
    G.st.view("g", 9)[17] = float("inf")
    lr = f32(L.hyper.lr)
    G.step(2, lr, _hyper(L.hyper, grad_norm=True))
    st = G.plan.query(clear=True)
    assert st & B.LAMB_STATUS_GRAD_NONFINITE
    assert not st & B.LAMB_STATUS_SKIPPED
    gn, gg, nf = _grad_norms(G)
    assert nf == 1 and math.isinf(gn[9]) and math.isinf(gg)
    assert all(math.isfinite(gn[k]) for k in range(L.n_tensors) if k != 9)
    # the step was applied (Inf/NaN propagate as in the plain step)
    assert not np.isfinite(G.download("w", 9)).all()
    G.close()


def test_huge_finite_gradient_saturates_the_norm_but_is_not_nonfinite():
    # |g| = 2^100: g^2 overflows fp32 in the chunk sums (the documented
    # limit of the fp32 partials), yet no element is Inf or NaN
    L = _layout()
    G = _prepared(L)
    G.st.view("g", 8)[5] = 2.0 ** 100
    G.step(2, f32(L.hyper.lr), _hyper(L.hyper, skip_nonfinite=True))
    st = G.plan.query(clear=True)
    assert not st & (B.LAMB_STATUS_GRAD_NONFINITE | B.LAMB_STATUS_SKIPPED)
    gn, gg, nf = _grad_norms(G)
    assert nf == 0 and math.isinf(gn[8]) and math.isinf(gg)
    assert int(G.d_step.item()) == 2           # step applied, no increment
    G.close()


# ---------------------------------------------------------------------------
# Skip on non-finite
# ---------------------------------------------------------------------------

def _with_flags(G, kind, h, lr, t, **flags):
    G.d_step.fill_(t)
    G.d_lr.fill_(lr)
    if kind == "lars":
        G.plan.lars_step(_hyper(h, True, **flags), G.d_step, G.d_lr)
    elif kind == "lamb":
        G.plan.lamb_step(_hyper(h, **flags), G.d_step, G.d_lr)
    else:
        G.plan.nlamb_step(_hyper(h, **flags), 0.004, kind == "nnlamb",
                          G.d_step, G.d_lr, G.d_prod)


KINDS = ["lamb", "nlamb", "nnlamb", "lars"]


@pytest.mark.parametrize("kind", KINDS)
@pytest.mark.parametrize("grad_dtype,copy_dtype", [("f32", None),
                                                    ("bf16", "bf16")])
def test_skip_mode_finite_step_is_bitwise_plain_step(kind, grad_dtype,
                                                     copy_dtype):
    L = _layout(grad_dtype, copy_dtype)
    lars = kind == "lars"
    h = W.Hyper(lr=0.5, trust_coef=1e-3, weight_decay=1e-4,
                bias_correction=False) if lars else L.hyper
    lr = f32(h.lr)
    runs = []
    for flags in ({}, {"skip_nonfinite": True}):
        G = _prepared(L, with_v=not lars)
        G.d_prod = torch.full((1,), 0.5, dtype=torch.float64, device="cuda:0")
        _with_flags(G, kind, h, lr, 2, increment_step=True, **flags)
        runs.append((_state(G), G.results()[0], int(G.d_step.item()),
                     float(G.d_prod.item())))
        G.close()
    (s0, r0, t0, p0), (s1, r1, t1, p1) = runs
    assert _bitwise_equal(s0, s1)
    assert np.array_equal(r0, r1) and t0 == t1 == 3 and p0 == p1


@pytest.mark.parametrize("kind", KINDS)
@pytest.mark.parametrize("bad", [float("nan"), float("inf"), -float("inf")])
def test_skip_mode_nonfinite_step_writes_nothing(kind, bad):
    L = _layout("bf16", "bf16")
    lars = kind == "lars"
    h = W.Hyper(lr=0.5, trust_coef=1e-3, weight_decay=1e-4,
                bias_correction=False) if lars else L.hyper
    G = _prepared(L, with_v=not lars)
    G.d_prod = torch.full((1,), 0.5, dtype=torch.float64, device="cuda:0")
    G.st.view("g", 12)[99999] = bad
    before = _state(G)
    sched = (1e-3, 10, 100)
    _with_flags(G, kind, h, 0.25, 2, increment_step=True,
                skip_nonfinite=True, lr_schedule=sched)
    st = G.plan.query(clear=True)
    assert st & B.LAMB_STATUS_SKIPPED and st & B.LAMB_STATUS_GRAD_NONFINITE
    assert _bitwise_equal(_state(G), before)
    assert int(G.d_step.item()) == 2               # t not advanced
    assert float(G.d_lr.item()) == 0.25            # eta_t not written
    assert float(G.d_prod.item()) == 0.5           # mu product unchanged
    assert _grad_norms(G)[2] == 1
    # repair the gradient: the next step is applied and matches the oracle
    G.load_grads(2, ks=[12])
    _with_flags(G, kind, h, 0.25, 2, increment_step=True,
                skip_nonfinite=True, lr_schedule=sched)
    assert G.plan.query() == 0 and int(G.d_step.item()) == 3
    assert _grad_norms(G)[2] == 0
    lr = f32(O.lr_schedule(2, *sched))
    ratio = G.results()[0]
    for k in range(L.n_tensors):
        w, g = L.weights(k), L.grad(k, 2)
        m, v = L.state_warm(k)
        lam = h.weight_decay * L.decay[k]
        g64 = O.to_f64(g, "bf16")
        if kind == "lars":
            ref = O.lars_tensor(w, g, m, lr=lr, decay=bool(L.decay[k]),
                                g_dtype="bf16", **hyper_kwargs(h, lars=True))
            compare_lars(G.download("w", k), G.download("m", k), ref, w, m,
                         g64, h.beta1, lam, TOL_STEP, lr=lr)
        elif kind == "lamb":
            ref = O.lamb_tensor(w, g, m, v, t=2, lr=lr, decay=bool(L.decay[k]),
                                g_dtype="bf16", **hyper_kwargs(h))
            compare_lamb(G.download("w", k), G.download("m", k),
                         G.download("v", k), ref, w, m, g64, h.beta1,
                         TOL_STEP, upd=(h, 2, lr, lam))
        else:
            ref = O.nlamb_tensor(w, g, m, v, t=2, lr=lr, mu_product=0.5,
                                 beta1=h.beta1, beta2=h.beta2, eps=h.eps,
                                 psi=0.004, weight_decay=h.weight_decay,
                                 decay=bool(L.decay[k]),
                                 nesterov_second_moment=kind == "nnlamb",
                                 phi_kind=h.phi, gamma_l=h.gamma_l,
                                 gamma_u=h.gamma_u, g_dtype="bf16")
            compare_nlamb(G.download("w", k), G.download("m", k),
                          G.download("v", k), ref, w, m, g64, h, 2, lr, lam,
                          0.004, 0.5, kind == "nnlamb", TOL_STEP)
        assert ratio_ok(ratio[k], ref.ratio), (kind, k)
    G.close()


def test_skip_decision_is_taken_on_the_device_inside_a_graph():
    """One captured step, replayed with finite, then non-finite, then
    finite gradients: the replay in the middle writes nothing."""
    L = _layout("bf16", "bf16")
    h = L.hyper
    G = _prepared(L)
    G.d_step.fill_(2)
    G.d_lr.fill_(f32(h.lr))
    hyp = _hyper(h, increment_step=True, skip_nonfinite=True)
    stream = torch.cuda.Stream()
    stream.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(stream):            # warm-up outside capture
        G.plan.lamb_step(hyp, G.d_step, G.d_lr, stream=stream)
    torch.cuda.current_stream().wait_stream(stream)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        G.plan.lamb_step(hyp, G.d_step, G.d_lr, stream=stream)
    torch.cuda.synchronize()
    G.plan.query(clear=True)
    t0 = int(G.d_step.item())
    graph.replay()
    torch.cuda.synchronize()
    assert int(G.d_step.item()) == t0 + 1 and G.plan.query() == 0
    G.st.view("g", 9)[3] = float("nan")
    snap = _state(G)
    graph.replay()
    torch.cuda.synchronize()
    assert _bitwise_equal(_state(G), snap)
    assert int(G.d_step.item()) == t0 + 1
    assert G.plan.query(clear=True) & B.LAMB_STATUS_SKIPPED
    G.load_grads(2, ks=[9])
    graph.replay()
    torch.cuda.synchronize()
    assert int(G.d_step.item()) == t0 + 2 and G.plan.query() == 0
    assert not _bitwise_equal(_state(G), snap)
    G.close()


# ---------------------------------------------------------------------------
# Decoupled weight decay
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("grad_dtype,copy_dtype", [("f32", None),
                                                    ("bf16", "bf16")])
@pytest.mark.parametrize("kind", ["lamb", "nlamb", "nnlamb"])
@pytest.mark.parametrize("algo", [1, 3], ids=["two_pass", "on_chip"])
def test_decoupled_decay_matches_oracle(grad_dtype, copy_dtype, kind, algo):
    L = _layout(grad_dtype, copy_dtype)
    h = W.Hyper(lr=2e-3, weight_decay=0.05, phi="clip", gamma_u=10.0)
    G = _prepared(L, algorithm=algo)
    G.d_prod = torch.full((1,), 0.5, dtype=torch.float64, device="cuda:0")
    lr = f32(h.lr)
    _with_flags(G, kind, h, lr, 2, decoupled_decay=True)
    ratio, wn, un = G.results()
    for k in range(L.n_tensors):
        w, g = L.weights(k), L.grad(k, 2)
        m, v = L.state_warm(k)
        g64 = O.to_f64(g, grad_dtype)
        if kind == "lamb":
            ref = O.lamb_tensor(w, g, m, v, t=2, lr=lr, decay=bool(L.decay[k]),
                                g_dtype=grad_dtype, decoupled_decay=True,
                                **hyper_kwargs(h))
            e = compare_lamb(G.download("w", k), G.download("m", k),
                             G.download("v", k), ref, w, m, g64, h.beta1,
                             TOL_STEP, upd=(h, 2, lr, 0.0))
        else:
            ref = O.nlamb_tensor(w, g, m, v, t=2, lr=lr, mu_product=0.5,
                                 beta1=h.beta1, beta2=h.beta2, eps=h.eps,
                                 psi=0.004, weight_decay=h.weight_decay,
                                 decay=bool(L.decay[k]),
                                 nesterov_second_moment=kind == "nnlamb",
                                 phi_kind=h.phi, gamma_l=h.gamma_l,
                                 gamma_u=h.gamma_u, g_dtype=grad_dtype,
                                 decoupled_decay=True)
            e = compare_nlamb(G.download("w", k), G.download("m", k),
                              G.download("v", k), ref, w, m, g64, h, 2, lr,
                              0.0, 0.004, 0.5, kind == "nnlamb", TOL_STEP)
        if copy_dtype:
            check_copy(G.download("copy", k), G.download("w", k), ref.w,
                       sw=e["_sw"])
        assert ratio_ok(ratio[k], ref.ratio), (k, ratio[k], ref.ratio)
        assert ratio_ok(un[k], ref.unorm), (k, un[k], ref.unorm)
    G.close()


def test_decoupled_decay_bert_large_sampled():
    """BERT-large at full size with decoupled decay: every tensor's trust
    ratio and ||r||, and a sample of tensors element by element."""
    L = W.bert_large_layout()
    h = L.hyper
    t = 1000
    lr = f32(h.lr)
    G = _prepared(L, step=t)
    G.d_step.fill_(t)
    G.d_lr.fill_(lr)
    G.plan.lamb_step(_hyper(h, decoupled_decay=True), G.d_step, G.d_lr)
    ratio, wn, un = G.results()
    full = set(range(0, L.n_tensors, 13)) | {0, L.n_tensors - 1}

    def check(k):
        w, g = L.weights(k), L.grad(k, t)
        m, v = L.state_warm(k)
        ref = O.lamb_tensor(w, g, m, v, t=t, lr=lr, decay=bool(L.decay[k]),
                            g_dtype="bf16", decoupled_decay=True,
                            **hyper_kwargs(h))
        assert ratio_ok(ratio[k], ref.ratio), (k, ratio[k], ref.ratio)
        assert ratio_ok(un[k], ref.unorm), k
        if k in full:
            e = compare_lamb(G.download("w", k), G.download("m", k),
                             G.download("v", k), ref, w, m,
                             O.to_f64(g, "bf16"), h.beta1, TOL_STEP,
                             upd=(h, t, lr, 0.0))
            check_copy(G.download("copy", k), G.download("w", k), ref.w,
                       sw=e["_sw"])

    oracle_map(check, range(L.n_tensors))
    G.close()


def test_decoupled_decay_rejected_for_lars():
    L = _layout()
    G = GpuLayout(L, with_v=False)
    with pytest.raises(B.LambError) as ei:
        G.plan.lars_step(_hyper(L.hyper, True, decoupled_decay=True),
                         G.d_step, G.d_lr)
    assert ei.value.status == B.LAMB_ERR_INVALID_ARG
    assert "DECOUPLED" in B.lamb_last_error()
    G.close()
