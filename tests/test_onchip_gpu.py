"""GPU parity of the on-chip single-touch step (LAMB_ALGO_ON_CHIP) against the
fp64 oracle, on grids and shared-memory sizes small enough that the edge
layout needs several resident rounds, pieces split across CTAs and streamed
tensors; plus its agreement with the two-pass kernels, its determinism, and
the bounded wait for the other CTAs' partial sums giving up (a wait made to
run out on purpose: nothing faults, the launch returns with
LAMB_STATUS_WAIT_TIMEOUT)."""
import math

import numpy as np
import pytest
import torch

from gpu_util import (TOL_RATIO, TOL_STEP, GpuLayout, c_hyper, check_copy,
                      compare_lamb, compare_lars, compare_nlamb, f32,
                      hyper_kwargs, ratio_ok)
from oracle import lamb_oracle as O
from paper_1904_00962_gb300 import binding as B
from paper_1904_00962_gb300 import build as build_mod
from paper_1904_00962_gb300 import workloads as W
from paper_1904_00962_gb300.state import LambPlan

pytestmark = pytest.mark.gpu

ON_CHIP = B.LAMB_ALGO_ON_CHIP
EDGE_SIZES = [0, 1, 2, 3, 4, 5, 7, 127, 128, 129, 1023, 1024, 1025, 16383,
              16384, 16385, 65539, 0, 3000, 100003, 256]
# (max CTAs, rows per CTA): the device's own sizes, then grids whose rounds
# hold 4096, 768 and 128 elements
GRIDS = [(0, 0), (8, 4), (3, 2), (1, 1)]


@pytest.fixture(scope="module", autouse=True)
def _lib(gpu):
    build_mod.build()
    B.load()
    yield
    torch.cuda.empty_cache()


def _layout(grad_dtype="f32", copy_dtype=None):
    n = len(EDGE_SIZES)
    return W.Layout(name="onchip_edge", names=[f"e{i}" for i in range(n)],
                    shapes=[(s,) for s in EDGE_SIZES],
                    decay=[i % 2 for i in range(n)],
                    init=[("normal", 0.02)] * n,
                    grad_sigma=[10 ** (-2 - (i % 4)) for i in range(n)],
                    grad_dtype=grad_dtype, copy_dtype=copy_dtype,
                    zero_w={3, 11}, zero_g={4, 12},
                    hyper=W.Hyper(lr=2e-3, phi="clip", gamma_l=0.0,
                                  gamma_u=10.0))


def _prepared(L, step, **kw):
    G = GpuLayout(L, algorithm=ON_CHIP, **kw)
    G.load_weights()
    G.load_warm_state()
    G.load_grads(step)
    return G


def _expected_streamed(sizes, info):
    cap = info["grid_blocks"] * info["rows_per_cta"]
    return sum(1 for s in sizes if (s + 127) // 128 > cap)


@pytest.mark.parametrize("grad_dtype,copy_dtype", [("f32", None),
                                                    ("bf16", "bf16")])
@pytest.mark.parametrize("misalign", [False, True])
@pytest.mark.parametrize("ctas,rows", GRIDS,
                         ids=[f"ctas{c}_rows{r}" for c, r in GRIDS])
def test_onchip_lamb_and_lars_edge_layout(grad_dtype, copy_dtype, misalign,
                                          ctas, rows):
    L = _layout(grad_dtype, copy_dtype)
    for lars in (False, True):
        h = (W.Hyper(lr=0.5, trust_coef=1e-3, weight_decay=1e-4,
                     bias_correction=False) if lars else L.hyper)
        G = _prepared(L, 3, with_v=not lars, onchip_max_ctas=ctas,
                      onchip_rows=rows,
                      misalign={5, 9, 13, 19} if misalign else None)
        info = G.plan.info()
        assert info["algorithm"] == ON_CHIP
        assert info["n_streamed_tensors"] == _expected_streamed(L.sizes, info)
        if rows:
            assert info["rows_per_cta"] == rows and info["n_rounds"] >= 2
        lr = f32(h.lr)
        G.step(3, lr, c_hyper(h, lars=lars), lars=lars)
        ratio, wn, un = G.results()
        for k in range(L.n_tensors):
            w, g = L.weights(k), L.grad(k, 3)
            m, v = L.state_warm(k)
            g64 = O.to_f64(g, grad_dtype)
            if lars:
                ref = O.lars_tensor(w, g, m, lr=lr, decay=bool(L.decay[k]),
                                    g_dtype=grad_dtype,
                                    **hyper_kwargs(h, lars=True))
                e = compare_lars(G.download("w", k), G.download("m", k), ref,
                                 w, m, g64, h.beta1,
                                 h.weight_decay * L.decay[k], TOL_STEP, lr=lr)
            else:
                ref = O.lamb_tensor(w, g, m, v, t=3, lr=lr,
                                    decay=bool(L.decay[k]), g_dtype=grad_dtype,
                                    **hyper_kwargs(h))
                e = compare_lamb(G.download("w", k), G.download("m", k),
                                 G.download("v", k), ref, w, m, g64, h.beta1,
                                 TOL_STEP,
                                 upd=(h, 3, lr, h.weight_decay * L.decay[k]))
            if copy_dtype:
                check_copy(G.download("copy", k), G.download("w", k), ref.w,
                           sw=e["_sw"])
            assert ratio_ok(ratio[k], ref.ratio), (lars, k, ratio[k],
                                                   ref.ratio)
            assert ratio_ok(wn[k], ref.wnorm), (lars, k)
            assert ratio_ok(un[k], ref.unorm), (lars, k)
            if L.sizes[k] == 0:
                assert ratio[k] == 1.0 and wn[k] == 0.0 and un[k] == 0.0
        G.close()


@pytest.mark.parametrize("nn", [False, True], ids=["nlamb", "nnlamb"])
@pytest.mark.parametrize("ctas,rows", [(0, 0), (8, 4)],
                         ids=["device", "ctas8_rows4"])
def test_onchip_nlamb_edge_layout(nn, ctas, rows):
    L = _layout("bf16", "bf16")
    h = L.hyper
    psi, prod, t = 0.004, 0.6, 5
    G = _prepared(L, t, onchip_max_ctas=ctas, onchip_rows=rows)
    d_prod = torch.full((1,), prod, dtype=torch.float64, device="cuda:0")
    lr = f32(h.lr)
    G.d_step.fill_(t)
    G.d_lr.fill_(lr)
    G.plan.nlamb_step(c_hyper(h, increment=True), psi, nn, G.d_step, G.d_lr,
                      d_prod)
    ratio, _, un = G.results()
    assert int(G.d_step.item()) == t + 1
    mu_t = O.nadam_mu(t, h.beta1, psi)
    assert math.isclose(float(d_prod.item()), prod * mu_t, rel_tol=1e-15)
    for k in range(L.n_tensors):
        w, g = L.weights(k), L.grad(k, t)
        m, v = L.state_warm(k)
        ref = O.nlamb_tensor(w, g, m, v, t=t, lr=lr, mu_product=prod,
                             beta1=h.beta1, beta2=h.beta2, eps=h.eps, psi=psi,
                             weight_decay=h.weight_decay,
                             decay=bool(L.decay[k]), nesterov_second_moment=nn,
                             phi_kind=h.phi, gamma_l=h.gamma_l,
                             gamma_u=h.gamma_u, g_dtype="bf16")
        e = compare_nlamb(G.download("w", k), G.download("m", k),
                          G.download("v", k), ref, w, m, O.to_f64(g, "bf16"),
                          h, t, lr, h.weight_decay * L.decay[k], psi, prod, nn,
                          TOL_STEP)
        check_copy(G.download("copy", k), G.download("w", k), ref.w,
                   sw=e["_sw"])
        assert ratio_ok(ratio[k], ref.ratio), (k, ratio[k], ref.ratio)
        assert ratio_ok(un[k], ref.unorm), k
    G.close()


@pytest.mark.parametrize("ctas,rows", [(0, 0), (8, 4)],
                         ids=["device", "ctas8_rows4"])
def test_onchip_decoupled_decay_and_schedule(ctas, rows):
    """Decoupled weight decay and the on-device learning-rate schedule on the
    on-chip kernel, against the oracle; the scheduled eta_t is written back
    and t advanced."""
    L = _layout()
    h = W.Hyper(lr=2e-3, weight_decay=0.05, phi="clip", gamma_u=10.0)
    t, base, warm, total = 7, 4e-3, 10, 100
    G = _prepared(L, t, onchip_max_ctas=ctas, onchip_rows=rows)
    G.d_step.fill_(t)
    hyp = B.make_hyper(beta1=h.beta1, beta2=h.beta2, eps=h.eps,
                       weight_decay=h.weight_decay, phi=h.phi,
                       gamma_l=h.gamma_l, gamma_u=h.gamma_u,
                       increment_step=True, decoupled_decay=True,
                       lr_schedule=(base, warm, total))
    G.plan.lamb_step(hyp, G.d_step, G.d_lr)
    lr = f32(O.lr_schedule(t, base, warm, total))
    assert float(G.d_lr.item()) == lr
    assert int(G.d_step.item()) == t + 1
    ratio, _, un = G.results()
    for k in range(L.n_tensors):
        w, g = L.weights(k), L.grad(k, t)
        m, v = L.state_warm(k)
        ref = O.lamb_tensor(w, g, m, v, t=t, lr=lr, decay=bool(L.decay[k]),
                            decoupled_decay=True, **hyper_kwargs(h))
        compare_lamb(G.download("w", k), G.download("m", k),
                     G.download("v", k), ref, w, m, g.astype(np.float64),
                     h.beta1, TOL_STEP, upd=(h, t, lr, 0.0))
        assert ratio_ok(ratio[k], ref.ratio), (k, ratio[k], ref.ratio)
        assert ratio_ok(un[k], ref.unorm), k
    G.close()


@pytest.mark.parametrize("name", ["bert_base", "resnet50"])
def test_onchip_matches_two_pass(name):
    """The moments do not depend on any reduction: bitwise equal to the
    two-pass kernels'.  The trust ratios differ only by the summation tree
    of the norms; w follows within the one-step tolerance."""
    L = W.get_layout(name)
    h = L.hyper
    outs = []
    for algo in (B.LAMB_ALGO_TWO_PASS, ON_CHIP):
        G = GpuLayout(L, algorithm=algo)
        G.load_weights()
        G.load_warm_state()
        G.load_grads(4)
        w_before = G.st.w.clone()
        G.step(4, f32(h.lr), c_hyper(h))
        r, _, _ = G.results()
        torch.cuda.synchronize()
        outs.append((G.st.w.clone(), G.st.m.clone(), G.st.v.clone(), r))
        G.close()
    (w1, m1, v1, r1), (w2, m2, v2, r2) = outs
    assert torch.equal(m1, m2) and torch.equal(v1, v2)
    np.testing.assert_allclose(r2, r1, rtol=2 * TOL_RATIO, atol=0)
    d = (w1.double() - w2.double()).abs()
    scale = torch.maximum(w1.double().abs(), w_before.double().abs())
    assert bool(torch.all(d <= TOL_STEP * scale))


@pytest.mark.parametrize("lars", [False, True])
def test_onchip_bitwise_repeatable(lars):
    """The partial sums have the plan's fixed shape: two plans of the same
    shape give the same bits, step after step."""
    L = W.resnet50_layout()
    h = L.lars_hyper if lars else L.hyper
    snaps = []
    for _ in range(2):
        G = _prepared(L, 4, with_v=not lars)
        for t in (4, 5, 6):
            G.step(t, f32(h.lr), c_hyper(h, lars=lars), lars=lars)
        torch.cuda.synchronize()
        snaps.append([G.st.w.clone(), G.st.m.clone()] +
                     list(G.plan.results()))
        assert G.plan.query() == 0
        G.close()
    for a, b in zip(*snaps):
        assert torch.equal(a, b)


def test_onchip_wait_gives_up_and_a_new_plan_works():
    """A plan whose CTAs wait for partial sums tagged for a launch that never
    comes (a test-only option): the first wait runs out after 20 ms, every
    CTA returns, the status word says LAMB_STATUS_WAIT_TIMEOUT, the context
    stays usable, later steps of that plan do nothing, and a new plan on the
    same state computes the step correctly."""
    L = _layout()
    h = L.hyper
    lr = f32(h.lr)
    # 4 CTAs with the device's rows: every tensor fits a round (none is
    # left to the two-pass kernels), and the layout takes two rounds
    G = _prepared(L, 2, test_unmet_wait=True, wait_limit_ms=20,
                  onchip_max_ctas=4)
    info = G.plan.info()
    assert info["n_streamed_tensors"] == 0 and info["n_rounds"] >= 2
    w0 = G.st.w.clone()
    G.step(2, lr, c_hyper(h))
    torch.cuda.synchronize()                 # the launch returned
    st = G.plan.query(clear=True)
    assert st & B.LAMB_STATUS_WAIT_TIMEOUT
    # the launch gave up at its first exchange: only round 0's pass 1 ran,
    # so no weight changed
    assert torch.equal(G.st.w, w0)
    G.load_warm_state()
    G.step(2, lr, c_hyper(h))                # an aborted plan does nothing
    torch.cuda.synchronize()
    assert torch.equal(G.st.w, w0)
    assert G.plan.query() == 0               # and sets no new status
    G.plan.destroy()
    G.plan = LambPlan(G.st, L.decay, algorithm=ON_CHIP, onchip_max_ctas=4)
    G.load_warm_state()
    G.step(2, lr, c_hyper(h))
    ratio, _, _ = G.results()
    for k in range(L.n_tensors):
        w, g = L.weights(k), L.grad(k, 2)
        m, v = L.state_warm(k)
        ref = O.lamb_tensor(w, g, m, v, t=2, lr=lr, decay=bool(L.decay[k]),
                            **hyper_kwargs(h))
        compare_lamb(G.download("w", k), G.download("m", k),
                     G.download("v", k), ref, w, m, g.astype(np.float64),
                     h.beta1, TOL_STEP,
                     upd=(h, 2, lr, h.weight_decay * L.decay[k]))
        assert ratio_ok(ratio[k], ref.ratio), k
    G.close()


def test_auto_picks_on_chip_unless_a_tensor_is_streamed():
    """LAMB_ALGO_AUTO: the on-chip step when no tensor is larger than a round
    (the tiny MLP, one round; ResNet-50, several), the two-pass step
    otherwise (BERT-base: its word embedding exceeds a round).  On ResNet-50,
    lamb_step runs the on-chip kernel (one launch) and lars_step the two
    two-pass kernels."""
    for name, want in (("mlp", ON_CHIP), ("resnet50", ON_CHIP),
                       ("bert_base", B.LAMB_ALGO_TWO_PASS)):
        L = W.get_layout(name)
        G = GpuLayout(L, algorithm=B.LAMB_ALGO_AUTO)
        info = G.plan.info()
        assert info["algorithm"] == want, name
        if want == ON_CHIP:
            assert info["n_streamed_tensors"] == 0
            # the host planner gives the same rounds for the device's grid
            _, rounds = B.lamb_layout_rounds(L.sizes, info["grid_blocks"],
                                             info["rows_per_cta"])
            assert info["n_rounds"] == rounds
            assert rounds == 1 if name == "mlp" else rounds > 1
        if name == "resnet50":
            G.load_weights()
            G.load_warm_state()
            G.load_grads(2)
            h = L.hyper
            for lars, launches in ((False, 1), (True, 2)):
                B.lamb_plan_set_timing(G.plan.handle, True)
                G.step(2, f32(h.lr), c_hyper(h, lars=lars), lars=lars)
                n, ms = B.lamb_plan_read_timing(G.plan.handle, 3)
                B.lamb_plan_set_timing(G.plan.handle, False)
                assert n == 1 and sum(x > 0 for x in ms) == launches, (lars, ms)
            assert G.plan.query(clear=True) == 0
        G.close()


@pytest.mark.parametrize("n,want", [(20, ON_CHIP), (40, B.LAMB_ALGO_TWO_PASS)])
def test_auto_takes_two_pass_beyond_32_rounds(n, want):
    """AUTO's round limit: with 4 CTAs of 8 rows (4,096 elements a round),
    n tensors of 4,000 elements take n rounds; 20 stay on-chip, 40 do not."""
    L = W.Layout(name="rounds", names=[f"t{i}" for i in range(n)],
                 shapes=[(4000,)] * n, decay=[1] * n,
                 init=[("normal", 0.02)] * n, grad_sigma=[1e-3] * n)
    G = GpuLayout(L, algorithm=B.LAMB_ALGO_AUTO, onchip_max_ctas=4,
                  onchip_rows=8)
    info = G.plan.info()
    assert info["algorithm"] == want
    if want == ON_CHIP:
        assert info["n_rounds"] == n
    G.close()
