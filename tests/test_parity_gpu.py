"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle on
the same seeded inputs, element by element, for every workload at full size,
plus edge cases, determinism, graph replay, resume and device status."""
import math

import numpy as np
import pytest
import torch

from gpu_util import (ALGO_IDS, ALGOS, TOL_CHAIN, TOL_RATIO, TOL_STEP,
                      GpuLayout, c_hyper, compare_nlamb,
                      check_copy, compare_lamb, compare_lars, f32,
                      hyper_kwargs, oracle_map, ratio_ok, worst_of)
from oracle import lamb_oracle as O
from paper_1904_00962_gb300 import binding as B
from paper_1904_00962_gb300 import build as build_mod
from paper_1904_00962_gb300 import workloads as W
from paper_1904_00962_gb300.state import DeviceState, LambPlan

pytestmark = pytest.mark.gpu

algos = pytest.mark.parametrize("algo", ALGOS, ids=lambda a: ALGO_IDS[a])


@pytest.fixture(scope="module", autouse=True)
def _lib(gpu):
    build_mod.build()
    B.load()
    yield
    torch.cuda.empty_cache()


def _oracle_lamb(L, k, w, g, m, v, t, lr, h):
    return O.lamb_tensor(w, g, m, v, t=t, lr=lr, decay=bool(L.decay[k]),
                         g_dtype=L.grad_dtype, **hyper_kwargs(h))


def _oracle_lars(L, k, w, g, m, lr, h):
    return O.lars_tensor(w, g, m, lr=lr, decay=bool(L.decay[k]),
                         g_dtype=L.grad_dtype, **hyper_kwargs(h, lars=True))


# ---------------------------------------------------------------------------
# Tiny MLP: chained steps with fresh seeded gradients (10 and 100 steps)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("n_steps", [10, 100])
@pytest.mark.parametrize("bias_correction", [True, False])
@algos
def test_mlp_chained_lamb(n_steps, bias_correction, algo):
    L = W.mlp_layout()
    h = L.hyper
    h.bias_correction = bias_correction
    G = GpuLayout(L, algorithm=algo)
    G.load_weights()
    lr = f32(h.lr)
    state = [(L.weights(k).astype(np.float64), np.zeros(L.sizes[k]),
              np.zeros(L.sizes[k])) for k in range(L.n_tensors)]
    hyp = c_hyper(h)
    worst = 0.0
    path = [np.zeros(s) for s in L.sizes]
    mpath = [np.zeros(s) for s in L.sizes]
    for t in range(1, n_steps + 1):
        G.load_grads(t)
        G.step(t, lr, hyp)
        ratio, _, _ = G.results()
        tol = TOL_STEP if t == 1 else TOL_CHAIN
        for k in range(L.n_tensors):
            w0, m0, v0 = state[k]
            g = L.grad(k, t)
            ref = _oracle_lamb(L, k, w0, g, m0, v0, t, lr, h)
            path[k] += np.abs(ref.w - w0)
            mpath[k] = h.beta1 * mpath[k] + (1 - h.beta1) * np.abs(g)
            e = compare_lamb(G.download("w", k), G.download("m", k),
                             G.download("v", k), ref, w0, m0,
                             g.astype(np.float64), h.beta1, tol,
                             w_path=path[k], m_path=mpath[k],
                             upd=(h, t, lr, h.weight_decay * L.decay[k]))
            worst = max(worst, worst_of(e))
            rt = TOL_RATIO if t == 1 else TOL_CHAIN
            assert ratio_ok(ratio[k], ref.ratio, rt), (t, k, ratio[k], ref.ratio)
            state[k] = (ref.w, ref.m, ref.v)
    G.close()
    print(f"mlp {n_steps} steps worst scaled err {worst:.3e}")


@algos
def test_mlp_chained_lars_100(algo):
    L = W.mlp_layout()
    h = W.Hyper(lr=1.0, beta1=0.9, weight_decay=1e-4, trust_coef=1e-3,
                phi="identity", bias_correction=False)
    G = GpuLayout(L, with_v=False, algorithm=algo)
    G.load_weights()
    lr = f32(h.lr)
    state = [(L.weights(k).astype(np.float64), np.zeros(L.sizes[k]))
             for k in range(L.n_tensors)]
    hyp = c_hyper(h, lars=True)
    path = [np.zeros(s) for s in L.sizes]
    mpath = [np.zeros(s) for s in L.sizes]
    for t in range(1, 101):
        G.load_grads(t)
        G.step(t, lr, hyp, lars=True)
        ratio, _, _ = G.results()
        tol = TOL_STEP if t == 1 else TOL_CHAIN
        for k in range(L.n_tensors):
            w0, m0 = state[k]
            g = L.grad(k, t)
            ref = _oracle_lars(L, k, w0, g, m0, lr, h)
            lam = h.weight_decay * L.decay[k]
            path[k] += np.abs(ref.w - w0)
            mpath[k] = h.beta1 * mpath[k] + (1 - h.beta1) * (
                np.abs(g) + lam * np.abs(w0))
            compare_lars(G.download("w", k), G.download("m", k), ref, w0, m0,
                         g.astype(np.float64), h.beta1, lam, tol,
                         w_path=path[k], lr=lr, m_path=mpath[k])
            assert ratio_ok(ratio[k], ref.ratio,
                            TOL_RATIO if t == 1 else TOL_CHAIN)
            state[k] = (ref.w, ref.m)
    G.close()


# ---------------------------------------------------------------------------
# Full-size layouts: one step from a warm state, EVERY tensor checked
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("name,lars", [("bert_base", False),
                                       ("bert_large", False),
                                       ("resnet50", False),
                                       ("resnet50", True)])
@algos
def test_full_layout_one_step_every_tensor(name, lars, algo):
    L = W.get_layout(name)
    h = L.lars_hyper if lars else L.hyper
    t = h.measured_step or (h.warm_steps + 1)
    G = GpuLayout(L, with_v=not lars, algorithm=algo)
    G.load_weights()
    G.load_warm_state()
    G.load_grads(t)
    lr = f32(h.lr)
    G.step(t, lr, c_hyper(h, lars=lars), lars=lars)
    ratio, wn, un = G.results()

    def check(k):
        w = L.weights(k)
        g = L.grad(k, t)
        m, v = L.state_warm(k)
        g64 = O.to_f64(g, L.grad_dtype)
        if lars:
            ref = _oracle_lars(L, k, w, g, m, lr, h)
            e = compare_lars(G.download("w", k), G.download("m", k), ref, w,
                             m, g64, h.beta1, h.weight_decay * L.decay[k],
                             TOL_STEP, lr=lr)
        else:
            ref = _oracle_lamb(L, k, w, g, m, v, t, lr, h)
            e = compare_lamb(G.download("w", k), G.download("m", k),
                             G.download("v", k), ref, w, m, g64, h.beta1,
                             TOL_STEP,
                             upd=(h, t, lr, h.weight_decay * L.decay[k]))
        if L.copy_dtype:
            check_copy(G.download("copy", k), G.download("w", k), ref.w,
                       sw=e["_sw"])
        assert ratio_ok(ratio[k], ref.ratio), (k, ratio[k], ref.ratio)
        assert ratio_ok(wn[k], ref.wnorm) and ratio_ok(un[k], ref.unorm), k
        return abs(ratio[k] - ref.ratio) / max(abs(ref.ratio), 1e-300)

    errs = oracle_map(check, range(L.n_tensors))
    G.close()
    print(f"{name} lars={lars}: worst trust-ratio rel err {max(errs):.3e}")


# ---------------------------------------------------------------------------
# Full-size layouts: the configured warm-up trajectory (3 chained steps, then
# the measured step), on a sample of tensors
# ---------------------------------------------------------------------------

def _sample(L, big=6):
    small = [k for k, s in enumerate(L.sizes) if s < 65536]
    large = [k for k, s in enumerate(L.sizes) if s >= 65536]
    pick = [large[i] for i in np.linspace(0, len(large) - 1, big).astype(int)]
    return sorted(set(small) | set(pick))


@pytest.mark.parametrize("name,lars", [("bert_base", False),
                                       ("bert_large", False),
                                       ("resnet50", False),
                                       ("resnet50", True)])
@algos
def test_full_layout_warm_trajectory(name, lars, algo):
    L = W.get_layout(name)
    h = L.lars_hyper if lars else L.hyper
    ts = list(range(1, h.warm_steps + 1)) + [h.measured_step or
                                               h.warm_steps + 1]
    G = GpuLayout(L, with_v=not lars, algorithm=algo)
    G.load_weights()
    lr = f32(h.lr)
    ks = _sample(L)
    state = {k: (L.weights(k).astype(np.float64), np.zeros(L.sizes[k]),
                 np.zeros(L.sizes[k])) for k in ks}
    hyp = c_hyper(h, lars=lars)
    final = {}
    path = {k: np.zeros(L.sizes[k]) for k in ks}
    mpath = {k: np.zeros(L.sizes[k]) for k in ks}
    for i, t in enumerate(ts):
        G.load_grads(i + 1)
        G.step(t, lr, hyp, lars=lars)
        for k in ks:
            w0, m0, v0 = state[k]
            g = L.grad(k, i + 1)
            g64 = O.to_f64(g, L.grad_dtype)
            lam = h.weight_decay * L.decay[k]
            if lars:
                r = _oracle_lars(L, k, w0, g, m0, lr, h)
                mpath[k] = h.beta1 * mpath[k] + (1 - h.beta1) * (
                    np.abs(g64) + lam * np.abs(w0))
            else:
                r = _oracle_lamb(L, k, w0, g, m0, v0, t, lr, h)
                mpath[k] = h.beta1 * mpath[k] + (1 - h.beta1) * np.abs(g64)
            path[k] += np.abs(r.w - w0)
            final[k] = (w0, m0, v0, r, g)
            state[k] = (r.w, r.m, None if lars else r.v)
    ratio, _, _ = G.results()
    for k in ks:
        w0, m0, v0, ref, g = final[k]
        g64 = O.to_f64(g, L.grad_dtype)
        if lars:
            e = compare_lars(G.download("w", k), G.download("m", k), ref, w0,
                             m0, g64, h.beta1, h.weight_decay * L.decay[k],
                             TOL_STEP, w_path=path[k], lr=lr,
                             m_path=mpath[k])
        else:
            e = compare_lamb(G.download("w", k), G.download("m", k),
                             G.download("v", k), ref, w0, m0, g64, h.beta1,
                             TOL_STEP, w_path=path[k], m_path=mpath[k],
                             upd=(h, ts[-1], lr, h.weight_decay * L.decay[k]))
        if L.copy_dtype:
            check_copy(G.download("copy", k), G.download("w", k), ref.w,
                       sw=e["_sw"])
        assert ratio_ok(ratio[k], ref.ratio), (k, ratio[k], ref.ratio)
    G.close()


# ---------------------------------------------------------------------------
# Ragged stress layout at full size (10,000 tensors, ~2.7e9 parameters)
# ---------------------------------------------------------------------------

@algos
def test_ragged_full_size(algo):
    L = W.ragged_layout()
    h = L.hyper
    G = GpuLayout(L, algorithm=algo)
    st = G.st
    gen = torch.Generator(device="cuda:0")
    gen.manual_seed(20200101)
    st.w.normal_(0.0, 0.02, generator=gen)   # bulk inputs of the tensors
    st.g.normal_(0.0, 1e-3, generator=gen)   # checked by properties only
    for k in L.zero_w:
        st.view("w", k).zero_()
    for k in L.zero_g:
        st.view("g", k).zero_()
    rng = np.random.default_rng(7)
    sizes = np.array(L.sizes)
    ks = set(rng.choice(L.n_tensors, 1000, replace=False).tolist())
    ks |= set(np.argsort(sizes)[-3:].tolist()) | set(np.argsort(sizes)[:5].tolist())
    ks |= set(list(L.zero_w)[:10]) | set(list(L.zero_g)[:10])
    ks = sorted(int(k) for k in ks)
    G.load_weights(ks)
    G.load_grads(1, ks)
    w_before = st.w.clone()
    lr = f32(h.lr)
    G.step(1, lr, c_hyper(h))
    ratio, wn, un = G.results()
    status = G.plan.query(clear=True)
    assert status == 0

    def check(k):
        w, g = L.weights(k), L.grad(k, 1)
        z = np.zeros(L.sizes[k])
        ref = _oracle_lamb(L, k, w, g, z, z, 1, lr, h)
        compare_lamb(G.download("w", k), G.download("m", k),
                     G.download("v", k), ref, w, z, g.astype(np.float64),
                     h.beta1, TOL_STEP,
                     upd=(h, 1, lr, h.weight_decay * L.decay[k]))
        assert ratio_ok(ratio[k], ref.ratio), (k, ratio[k], ref.ratio)
        assert ratio_ok(wn[k], ref.wnorm) and ratio_ok(un[k], ref.unorm)
    oracle_map(check, ks)

    # every tensor: ||w' - w|| = eta * rho * ||u||, rho*||u|| = phi(||w||),
    # and ||w|| agrees with an independent fp64 reduction of the input
    for k in range(L.n_tensors):
        o, n = st.offsets[k], L.sizes[k]
        wb = w_before[o:o + n].double()
        d = float(torch.linalg.vector_norm(st.w[o:o + n].double() - wb))
        wnk = float(torch.linalg.vector_norm(wb))
        assert math.isclose(wn[k], wnk, rel_tol=1e-6, abs_tol=0), k
        if wn[k] == 0 or un[k] == 0:
            assert ratio[k] == 1.0, k
            assert math.isclose(d, lr * un[k], rel_tol=2e-3, abs_tol=1e-30), k
        else:
            phi = min(max(wn[k], h.gamma_l), h.gamma_u)
            # fp64 ratio (two-pass): exact to fp64 rounding;
            # the on-chip kernel forms rho = RN32(phi / ||u||) in fp32
            assert math.isclose(ratio[k] * un[k], phi,
                                rel_tol=2.5e-7 if algo == 3 else 1e-12), k
            assert math.isclose(d, lr * phi, rel_tol=2e-3), (k, d, lr * phi)
    for k in L.zero_w:
        assert ratio[k] == 1.0 and wn[k] == 0.0
    G.close()
    del w_before


# ---------------------------------------------------------------------------
# Edge cases: empty, 1-element, ragged tails, chunk boundaries, misaligned
# pointers (element-wise path), zero norms, several chunk sizes and grids,
# bf16 gradients with the bf16 copy, phi variants
# ---------------------------------------------------------------------------

EDGE_SIZES = [0, 1, 2, 3, 4, 5, 7, 1023, 1024, 1025, 16383, 16384, 16385,
              65539, 0, 3000, 100003]


def _edge_layout(grad_dtype="f32", copy_dtype=None, name="edge"):
    n = len(EDGE_SIZES)
    return W.Layout(name=name, names=[f"e{i}" for i in range(n)],
                    shapes=[(s,) for s in EDGE_SIZES],
                    decay=[i % 2 for i in range(n)],
                    init=[("normal", 0.02)] * n,
                    grad_sigma=[10 ** (-2 - (i % 4)) for i in range(n)],
                    grad_dtype=grad_dtype, copy_dtype=copy_dtype,
                    zero_w={3, 10}, zero_g={4, 11},
                    hyper=W.Hyper(lr=2e-3, phi="clip", gamma_l=0.0,
                                  gamma_u=10.0))


@pytest.mark.parametrize("grad_dtype,copy_dtype", [("f32", None),
                                                    ("bf16", "bf16"),
                                                    ("f32", "bf16")])
@pytest.mark.parametrize("chunk,bps", [(1024, 0), (0, 0), (65536, 1),
                                       (1024, 1)])
@pytest.mark.parametrize("misalign", [False, True])
def test_edge_layout(grad_dtype, copy_dtype, chunk, bps, misalign):
    L = _edge_layout(grad_dtype, copy_dtype)
    h = L.hyper
    G = GpuLayout(L, chunk_elems=chunk, blocks_per_sm=bps,
                  misalign={5, 9, 12, 16} if misalign else None)
    info = G.plan.info()
    if misalign:
        assert info["n_vector_tensors"] < L.n_tensors
    G.load_weights()
    G.load_warm_state()
    G.load_grads(2)
    lr = f32(h.lr)
    G.step(2, lr, c_hyper(h))
    ratio, wn, un = G.results()
    for k in range(L.n_tensors):
        w, g = L.weights(k), L.grad(k, 2)
        m, v = L.state_warm(k)
        ref = _oracle_lamb(L, k, w, g, m, v, 2, lr, h)
        e = compare_lamb(G.download("w", k), G.download("m", k),
                         G.download("v", k), ref, w, m,
                         O.to_f64(g, grad_dtype), h.beta1, TOL_STEP,
                         upd=(h, 2, lr, h.weight_decay * L.decay[k]))
        if copy_dtype:
            check_copy(G.download("copy", k), G.download("w", k), ref.w,
                       sw=e["_sw"])
        assert ratio_ok(ratio[k], ref.ratio), (k, ratio[k], ref.ratio)
        if L.sizes[k] == 0:
            assert ratio[k] == 1.0 and wn[k] == 0.0 and un[k] == 0.0
    G.close()


@pytest.mark.parametrize("phi,gl,gu", [("identity", 0.0, math.inf),
                                       ("clip", 0.5, 0.6),
                                       ("clip", 0.0, 1e-3)])
@algos
def test_edge_layout_phi_and_lars(phi, gl, gu, algo):
    L = _edge_layout()
    for lars in (False, True):
        h = W.Hyper(lr=0.5 if lars else 2e-3, phi=phi, gamma_l=gl, gamma_u=gu,
                    trust_coef=1e-3 if lars else 1.0, weight_decay=0.01,
                    bias_correction=not lars)
        G = GpuLayout(L, with_v=not lars, algorithm=algo)
        G.load_weights()
        G.load_warm_state()
        G.load_grads(3)
        lr = f32(h.lr)
        G.step(3, lr, c_hyper(h, lars=lars), lars=lars)
        ratio, _, _ = G.results()
        for k in range(L.n_tensors):
            w, g = L.weights(k), L.grad(k, 3)
            m, v = L.state_warm(k)
            if lars:
                ref = _oracle_lars(L, k, w, g, m, lr, h)
                compare_lars(G.download("w", k), G.download("m", k), ref, w,
                             m, g.astype(np.float64), h.beta1,
                             h.weight_decay * L.decay[k], TOL_STEP, lr=lr)
            else:
                ref = _oracle_lamb(L, k, w, g, m, v, 3, lr, h)
                compare_lamb(G.download("w", k), G.download("m", k),
                             G.download("v", k), ref, w, m,
                             g.astype(np.float64), h.beta1, TOL_STEP,
                             upd=(h, 3, lr, h.weight_decay * L.decay[k]))
            assert ratio_ok(ratio[k], ref.ratio), (lars, k)
        G.close()


# ---------------------------------------------------------------------------
# Determinism: bitwise equal across runs and across grid shapes
# ---------------------------------------------------------------------------

def _snapshot(G):
    torch.cuda.synchronize()
    out = [G.st.w.clone(), G.st.m.clone()]
    if G.st.v is not None:
        out.append(G.st.v.clone())
    if G.st.copy is not None:
        out.append(G.st.copy.clone())
    return out + [t.clone() for t in G.plan.results()]


@pytest.mark.parametrize("lars", [False, True])
def test_bitwise_deterministic_across_runs_and_grids(lars):
    L = W.resnet50_layout()
    h = L.lars_hyper if lars else L.hyper
    snaps = []
    for bps in (0, 1, 0):
        G = GpuLayout(L, with_v=not lars, blocks_per_sm=bps, chunk_elems=4096)
        G.load_weights()
        G.load_warm_state()
        G.load_grads(4)
        for t in (4, 5):
            G.step(t, f32(h.lr), c_hyper(h, lars=lars), lars=lars)
        snaps.append(_snapshot(G))
        G.close()
    for other in snaps[1:]:
        for a, b in zip(snaps[0], other):
            assert torch.equal(a.view(torch.uint8) if a.dtype == torch.bfloat16
                               else a, b.view(torch.uint8)
                               if b.dtype == torch.bfloat16 else b)


# ---------------------------------------------------------------------------
# CUDA graph capture: replays read eta and t from device memory
# ---------------------------------------------------------------------------

@algos
def test_graph_replay_equals_eager(algo):
    L = W.bert_layout(2, 128, 512, vocab=1000, positions=64, name="tinybert",
                      grad_dtype="bf16", copy_dtype="bf16")
    h = L.hyper
    lrs = [f32(x) for x in (1e-3, 2e-3, 5e-4, 3e-3, 1e-3)]
    hyp = c_hyper(h, increment=True)

    def fresh():
        G = GpuLayout(L, algorithm=algo)
        G.load_weights()
        G.d_step.fill_(1)
        return G

    eager = fresh()
    for i, lr in enumerate(lrs):
        eager.load_grads(i + 1)
        eager.d_lr.fill_(lr)
        eager.plan.lamb_step(hyp, eager.d_step, eager.d_lr)
    snap_e = _snapshot(eager)
    assert int(eager.d_step.item()) == 6

    G = fresh()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=s):
        G.plan.lamb_step(hyp, G.d_step, G.d_lr)
    torch.cuda.synchronize()
    assert int(G.d_step.item()) == 1          # capture ran nothing
    for i, lr in enumerate(lrs):
        G.load_grads(i + 1)
        G.d_lr.fill_(lr)
        graph.replay()
    snap_g = _snapshot(G)
    assert int(G.d_step.item()) == 6
    for a, b in zip(snap_e, snap_g):
        assert torch.equal(a.view(torch.int16) if a.dtype == torch.bfloat16
                           else a, b.view(torch.int16)
                           if b.dtype == torch.bfloat16 else b)
    eager.close()
    G.close()


@algos
@pytest.mark.parametrize("lars", [False, True], ids=["lamb", "lars"])
def test_step_call_equals_the_plain_binding(algo, lars):
    """binding.step_call marshals the arguments once; the steps it runs must
    be the ones lamb_step / lars_step run, bit for bit."""
    L = W.bert_layout(1, 64, 256, vocab=500, positions=32, name="stepcall")
    h = L.hyper
    hyp = c_hyper(h, increment=True, lars=lars)
    snaps = []
    for use_call in (False, True):
        G = GpuLayout(L, with_v=not lars, algorithm=algo)
        G.load_weights()
        G.load_warm_state()
        G.d_step.fill_(2)
        G.d_lr.fill_(f32(h.lr))
        call = G.plan.step_call("lars" if lars else "lamb", hyp, G.d_step,
                                G.d_lr)
        for t in (2, 3, 4):
            G.load_grads(t)
            if use_call:
                call()
            elif lars:
                G.plan.lars_step(hyp, G.d_step, G.d_lr)
            else:
                G.plan.lamb_step(hyp, G.d_step, G.d_lr)
        assert G.plan.query(clear=True) == 0
        assert int(G.d_step.item()) == 5
        snaps.append(_snapshot(G))
        G.close()
    for a, b in zip(*snaps):
        assert torch.equal(a, b)


# ---------------------------------------------------------------------------
# Checkpoint / resume: state is caller-owned, the plan is stateless
# ---------------------------------------------------------------------------

@algos
def test_split_run_resume_is_bitwise_equal(algo):
    L = W.bert_layout(1, 64, 256, vocab=500, positions=32, name="resume")
    h = L.hyper
    hyp = c_hyper(h, increment=True)

    def run(G, steps):
        for s in steps:
            G.load_grads(s)
            G.d_lr.fill_(f32(h.lr))
            G.plan.lamb_step(hyp, G.d_step, G.d_lr)

    full = GpuLayout(L, algorithm=algo)
    full.load_weights()
    run(full, range(1, 13))
    a = GpuLayout(L, algorithm=algo)
    a.load_weights()
    run(a, range(1, 7))
    torch.cuda.synchronize()
    ckpt = {n: getattr(a.st, n).cpu() for n in ("w", "m", "v")}
    step = a.d_step.cpu()
    a.close()
    b = GpuLayout(L, algorithm=algo)
    for n, t in ckpt.items():
        getattr(b.st, n).copy_(t)
    b.d_step.copy_(step)
    run(b, range(7, 13))
    torch.cuda.synchronize()
    for n in ("w", "m", "v"):
        assert torch.equal(getattr(full.st, n), getattr(b.st, n)), n
    assert int(b.d_step.item()) == 13
    full.close()
    b.close()


# ---------------------------------------------------------------------------
# Device-side status and argument handling
# ---------------------------------------------------------------------------

@algos
def test_bad_step_count_skips_step_and_sets_status(algo):
    L = W.mlp_layout()
    G = GpuLayout(L, algorithm=algo)
    G.load_weights()
    G.load_grads(1)
    before = _snapshot(G)[:3]
    hyp = c_hyper(L.hyper, increment=True)
    G.d_step.fill_(0)
    G.d_lr.fill_(1e-3)
    G.plan.lamb_step(hyp, G.d_step, G.d_lr)
    st = G.plan.query(clear=True)
    assert st & B.LAMB_STATUS_BAD_STEP
    after = _snapshot(G)[:3]
    for a, b in zip(before, after):
        assert torch.equal(a, b)
    assert int(G.d_step.item()) == 0
    # the plan still works afterwards
    G.d_step.fill_(1)
    G.plan.lamb_step(hyp, G.d_step, G.d_lr)
    assert G.plan.query() == 0
    assert int(G.d_step.item()) == 2
    r, _, _ = G.results()
    for k in range(L.n_tensors):
        z = np.zeros(L.sizes[k])
        ref = _oracle_lamb(L, k, L.weights(k), L.grad(k, 1), z, z, 1,
                           f32(1e-3), L.hyper)
        assert ratio_ok(r[k], ref.ratio)
    G.close()


@algos
def test_nonfinite_gradient_propagates_and_is_flagged(algo):
    L = _edge_layout()
    G = GpuLayout(L, algorithm=algo)
    G.load_weights()
    G.load_grads(1)
    bad = 9
    G.st.view("g", bad)[17] = float("nan")
    lr = f32(L.hyper.lr)
    G.step(1, lr, c_hyper(L.hyper))
    assert G.plan.query(clear=True) & B.LAMB_STATUS_NONFINITE
    ratio, _, _ = G.results()
    assert math.isnan(ratio[bad])
    for k in range(L.n_tensors):
        w, g = L.weights(k), L.grad(k, 1).copy()
        if k == bad:
            g[17] = np.nan
        z = np.zeros(L.sizes[k])
        ref = _oracle_lamb(L, k, w, g, z, z, 1, lr, L.hyper)
        compare_lamb(G.download("w", k), G.download("m", k),
                     G.download("v", k), ref, w, z, g.astype(np.float64),
                     L.hyper.beta1, TOL_STEP,
                     upd=(L.hyper, 1, lr, L.hyper.weight_decay * L.decay[k]))
        assert ratio_ok(ratio[k], ref.ratio)
    assert np.isnan(G.download("w", bad)).all()
    G.close()


@algos
def test_increment_step_matches_oracle_chain(algo):
    L = W.mlp_layout()
    h = L.hyper
    G = GpuLayout(L, algorithm=algo)
    G.load_weights()
    G.d_step.fill_(1)
    G.d_lr.fill_(f32(h.lr))
    hyp = c_hyper(h, increment=True)
    state = [(L.weights(k).astype(np.float64), np.zeros(L.sizes[k]),
              np.zeros(L.sizes[k])) for k in range(L.n_tensors)]
    path = [np.zeros(s) for s in L.sizes]
    for t in (1, 2, 3):
        G.load_grads(t)
        G.plan.lamb_step(hyp, G.d_step, G.d_lr)
        for k in range(L.n_tensors):
            w0, m0, v0 = state[k]
            r = _oracle_lamb(L, k, w0, L.grad(k, t), m0, v0, t, f32(h.lr), h)
            path[k] += np.abs(r.w - w0)
            state[k] = (r.w, r.m, r.v)
    torch.cuda.synchronize()
    assert int(G.d_step.item()) == 4
    for k in range(L.n_tensors):
        got = G.download("w", k).astype(np.float64)
        scale = np.maximum(np.abs(state[k][0]), path[k])
        assert np.all(np.abs(got - state[k][0]) <= TOL_STEP * scale)
    G.close()



@algos
def test_two_plans_alternating_gradient_buffers(algo):
    """Double-buffered gradients, the pattern of a training loop that
    uploads (or computes) step t+1's gradients while step t runs: two plans
    over the same w, m, v and bf16 copy, each bound to its own gradient
    buffer, take turns on one stream with one device step counter
    (INCREMENT_STEP).  Every step must equal, bit for bit, one plan stepping
    through the same gradients in a single buffer."""
    L = W.bert_layout(2, 256, 1024, name="bert_small", grad_dtype="bf16",
                      copy_dtype="bf16")
    h = L.hyper
    hyp = c_hyper(h, increment=True)
    dev = torch.device("cuda:0")
    gen = torch.Generator(device=dev)

    def grads(t, total):
        gen.manual_seed(1000 + t)
        return (torch.randn(total, device=dev, generator=gen) *
                1e-3).to(torch.bfloat16)

    def fresh():
        G = GpuLayout(L, algorithm=algo)
        G.load_weights()
        G.d_step.fill_(1)
        G.d_lr.fill_(f32(h.lr))
        return G

    n_steps = 6
    # one plan, one buffer
    A = fresh()
    ref = []
    for t in range(1, n_steps + 1):
        A.st.g.copy_(grads(t, A.st.total))
        A.plan.lamb_step(hyp, A.d_step, A.d_lr)
        r, _, _ = A.plan.results()
        ref.append(r.clone())
    torch.cuda.synchronize()
    # two plans, two buffers, alternating
    Bl = fresh()
    st = Bl.st
    g2 = torch.empty_like(st.g)
    plan2 = LambPlan(st, L.decay, algorithm=algo)
    es = st.g.element_size()
    B.lamb_plan_bind(plan2.handle, st.ptrs("w"),
                     [g2.data_ptr() + es * o for o in st.offsets],
                     st.ptrs("m"), st.ptrs("v"), st.ptrs("copy"))
    bufs, plans = [st.g, g2], [Bl.plan, plan2]
    for t in range(1, n_steps + 1):
        i = (t - 1) % 2
        bufs[i].copy_(grads(t, st.total))
        plans[i].lamb_step(hyp, Bl.d_step, Bl.d_lr)
        r, _, _ = plans[i].results()
        assert torch.equal(r, ref[t - 1]), t
    torch.cuda.synchronize()
    assert int(Bl.d_step.item()) == n_steps + 1 == int(A.d_step.item())
    assert plan2.query() == 0 and Bl.plan.query() == 0
    for name in ("w", "m", "v", "copy"):
        assert torch.equal(getattr(st, name), getattr(A.st, name)), name
    plan2.destroy()
    A.close()
    Bl.close()

def test_argument_errors_on_device_plans():
    L = W.mlp_layout()
    st = DeviceState(L.sizes, with_v=False)
    plan = LambPlan(st, L.decay)
    d_lr = torch.ones(1, device="cuda:0")
    with pytest.raises(B.LambError) as ei:             # no v bound
        plan.lamb_step(B.make_hyper(), torch.ones(1, dtype=torch.int64,
                                                  device="cuda:0"), d_lr)
    assert ei.value.status == B.LAMB_ERR_NOT_BOUND
    with pytest.raises(B.LambError) as ei:             # d_step needed
        B.lars_step(plan.handle, B.make_hyper(increment_step=True), 0,
                    d_lr.data_ptr())
    assert ei.value.status == B.LAMB_ERR_INVALID_ARG
    for bad in (dict(beta1=1.0), dict(phi="clip", gamma_l=2.0, gamma_u=1.0),
                dict(weight_decay=math.nan)):
        with pytest.raises(B.LambError):
            B.lars_step(plan.handle, B.make_hyper(**bad), 0, d_lr.data_ptr())
    with pytest.raises(B.LambError):                   # d_lr NULL
        B.lars_step(plan.handle, B.make_hyper(bias_correction=False), 0, 0)
    # LARS without a step counter is fine
    plan.lars_step(B.make_hyper(bias_correction=False, trust_coef=1e-3), None,
                   d_lr)
    torch.cuda.synchronize()
    # pointer misaligned below the element size
    with pytest.raises(B.LambError):
        B.lamb_plan_bind(plan.handle, [p + 1 for p in st.ptrs("w")],
                         st.ptrs("g"), st.ptrs("m"))
    info = plan.info()
    assert info["n_tensors"] == 4 and info["bound"] == 1
    assert info["num_sms"] > 0 and info["grid_blocks"] >= 1
    plan.destroy()


def test_non_default_stream_and_rebind():
    L = W.resnet50_layout()
    h = L.hyper
    A = GpuLayout(L)
    A.load_weights(); A.load_warm_state(); A.load_grads(4)
    B2 = DeviceState(L.sizes)
    for n in ("w", "m", "v", "g"):
        getattr(B2, n).copy_(getattr(A.st, n))
    A.step(4, f32(h.lr), c_hyper(h))
    ref = _snapshot(A)
    # same plan, rebound to the copy, run on a side stream
    A.plan.state = B2
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        A.plan.bind(stream=s)
        A.d_step.fill_(4)
        A.plan.lamb_step(c_hyper(h), A.d_step, A.d_lr, stream=s)
    torch.cuda.synchronize()
    assert torch.equal(B2.w, ref[0]) and torch.equal(B2.m, ref[1])
    assert torch.equal(B2.v, ref[2])
    r_ptr, w_ptr, u_ptr = B.lamb_plan_trust_ratios(A.plan.handle)
    assert r_ptr and w_ptr and u_ptr
    A.close()


@algos
def test_timing_hook_records_both_kernels(algo):
    L = W.resnet50_layout()
    G = GpuLayout(L, algorithm=algo)
    G.load_weights(); G.load_grads(1)
    B.lamb_plan_set_timing(G.plan.handle, True)
    for t in range(1, 4):
        G.step(t, f32(1e-3), c_hyper(L.hyper))
    n, ms = B.lamb_plan_read_timing(G.plan.handle, 2)
    assert n == 3 and ms[0] > 0
    assert (ms[1] > 0) if algo == 1 else (ms[1] == 0)
    assert G.plan.info()["algorithm"] == algo
    B.lamb_plan_set_timing(G.plan.handle, False)
    G.close()


# ---------------------------------------------------------------------------
# N-LAMB / NN-LAMB (appendix Algorithms 3 and 4)
# ---------------------------------------------------------------------------

def _oracle_nlamb(L, k, w, g, m, v, t, lr, h, prod, psi, nn):
    return O.nlamb_tensor(w, g, m, v, t=t, lr=lr, mu_product=prod,
                          beta1=h.beta1, beta2=h.beta2, eps=h.eps, psi=psi,
                          weight_decay=h.weight_decay, decay=bool(L.decay[k]),
                          nesterov_second_moment=nn, phi_kind=h.phi,
                          gamma_l=h.gamma_l, gamma_u=h.gamma_u,
                          g_dtype=L.grad_dtype)


@pytest.mark.parametrize("nn", [False, True], ids=["nlamb", "nnlamb"])
def test_nlamb_chained_mlp_and_edge(nn):
    """20 chained steps with the step counter and the momentum product
    advanced on the device, on the MLP and the edge-case layout."""
    psi = 0.004
    for L in (W.mlp_layout(), _edge_layout()):
        h = W.Hyper(lr=1e-3, beta1=0.975, beta2=0.999, eps=1e-8,
                    weight_decay=0.01, phi="clip", gamma_u=10.0)
        G = GpuLayout(L)
        G.load_weights()
        hyp = c_hyper(h, increment=True)
        d_prod = torch.ones(1, dtype=torch.float64, device="cuda:0")
        G.d_step.fill_(1)
        G.d_lr.fill_(f32(h.lr))
        lr = f32(h.lr)
        state = [(L.weights(k).astype(np.float64), np.zeros(s), np.zeros(s))
                 for k, s in enumerate(L.sizes)]
        path = [np.zeros(s) for s in L.sizes]
        mpath = [np.zeros(s) for s in L.sizes]
        prod = 1.0
        for t in range(1, 21):
            G.load_grads(t)
            G.plan.nlamb_step(hyp, psi, nn, G.d_step, G.d_lr, d_prod)
            ratio, _, _ = G.results()
            tol = TOL_STEP if t == 1 else TOL_CHAIN
            new_prod = None
            for k in range(L.n_tensors):
                w0, m0, v0 = state[k]
                g = L.grad(k, t)
                ref = _oracle_nlamb(L, k, w0, g, m0, v0, t, lr, h, prod, psi, nn)
                path[k] += np.abs(ref.w - w0)
                mpath[k] = h.beta1 * mpath[k] + (1 - h.beta1) * np.abs(g)
                compare_nlamb(G.download("w", k), G.download("m", k),
                              G.download("v", k), ref, w0, m0,
                              g.astype(np.float64), h, t, lr,
                              h.weight_decay * L.decay[k], psi, prod, nn, tol,
                              w_path=path[k], m_path=mpath[k])
                assert ratio_ok(ratio[k], ref.ratio,
                                TOL_RATIO if t == 1 else TOL_CHAIN), (t, k)
                state[k] = (ref.w, ref.m, ref.v)
                new_prod = ref.mu_product
            prod = new_prod
            assert math.isclose(float(d_prod.item()), prod, rel_tol=1e-14)
            assert int(G.d_step.item()) == t + 1
        G.close()


@pytest.mark.parametrize("nn", [False, True], ids=["nlamb", "nnlamb"])
def test_nlamb_bert_large_one_step_every_tensor(nn):
    """BERT-large layout (bf16 gradients, bf16 copy) at t = 1000 from a warm
    state, every tensor against the oracle."""
    L = W.bert_large_layout()
    h = W.Hyper(lr=2e-3, beta1=0.975, beta2=0.999, eps=1e-8,
                weight_decay=0.01, phi="clip", gamma_u=10.0)
    psi, t = 0.004, 1000
    prod = math.prod(O.nadam_mu(i, h.beta1, psi) for i in range(1, t))
    G = GpuLayout(L)
    G.load_weights()
    G.load_warm_state()
    G.load_grads(t)
    lr = f32(h.lr)
    d_prod = torch.full((1,), prod, dtype=torch.float64, device="cuda:0")
    G.d_step.fill_(t)
    G.d_lr.fill_(lr)
    G.plan.nlamb_step(c_hyper(h), psi, nn, G.d_step, G.d_lr, d_prod)
    ratio, wn, un = G.results()

    def check(k):
        w, g = L.weights(k), L.grad(k, t)
        m, v = L.state_warm(k)
        ref = _oracle_nlamb(L, k, w, g, m, v, t, lr, h, prod, psi, nn)
        e = compare_nlamb(G.download("w", k), G.download("m", k),
                          G.download("v", k), ref, w, m,
                          O.to_f64(g, L.grad_dtype), h, t, lr,
                          h.weight_decay * L.decay[k], psi, prod, nn, TOL_STEP)
        check_copy(G.download("copy", k), G.download("w", k), ref.w,
                   sw=e["_sw"])
        assert ratio_ok(ratio[k], ref.ratio), (k, ratio[k], ref.ratio)
        assert ratio_ok(wn[k], ref.wnorm) and ratio_ok(un[k], ref.unorm), k
        return ref.mu_product

    prods = oracle_map(check, range(L.n_tensors))
    assert math.isclose(float(d_prod.item()), prods[0], rel_tol=1e-14)
    G.close()


def test_nlamb_argument_errors():
    L = W.mlp_layout()
    G = GpuLayout(L)
    d_prod = torch.ones(1, dtype=torch.float64, device="cuda:0")
    h = c_hyper(L.hyper)
    with pytest.raises(B.LambError):          # negative momentum decay
        G.plan.nlamb_step(h, -1.0, False, G.d_step, G.d_lr, d_prod)
    with pytest.raises(B.LambError):          # product state required
        B.nlamb_step(G.plan.handle, h, 0.004, 0, G.d_step.data_ptr(),
                     G.d_lr.data_ptr(), 0)
    G.close()


# ---------------------------------------------------------------------------
# Section 4 learning-rate schedule computed on the device (reading Q16)
# ---------------------------------------------------------------------------

@algos
def test_lr_schedule_on_device(algo):
    L = W.mlp_layout()
    h = L.hyper
    eta0, tw, T = 4e-3, 4, 10
    G = GpuLayout(L, algorithm=algo)
    G.load_weights()
    hyp = B.make_hyper(beta1=h.beta1, beta2=h.beta2, eps=h.eps,
                       weight_decay=h.weight_decay, phi=h.phi,
                       increment_step=True, lr_schedule=(eta0, tw, T))
    G.d_step.fill_(1)
    state = [(L.weights(k).astype(np.float64), np.zeros(s), np.zeros(s))
             for k, s in enumerate(L.sizes)]
    path = [np.zeros(s) for s in L.sizes]
    for t in range(1, 13):
        G.load_grads(t)
        G.plan.lamb_step(hyp, G.d_step, G.d_lr)
        ratio, _, _ = G.results()
        lr = f32(O.lr_schedule(t, eta0, tw, T))
        assert float(G.d_lr.item()) == lr, t          # the eta_t it applied
        for k in range(L.n_tensors):
            w0, m0, v0 = state[k]
            ref = _oracle_lamb(L, k, w0, L.grad(k, t), m0, v0, t, lr, h)
            path[k] += np.abs(ref.w - w0)
            got = G.download("w", k).astype(np.float64)
            scale = np.maximum(np.maximum(np.abs(ref.w), np.abs(w0)), path[k])
            assert np.all(np.abs(got - ref.w) <= TOL_CHAIN * scale), (t, k)
            state[k] = (ref.w, ref.m, ref.v)
    assert int(G.d_step.item()) == 13
    # after T the schedule is 0: weights stop moving
    w_before = G.st.w.clone()
    G.load_grads(99)
    G.plan.lamb_step(hyp, G.d_step, G.d_lr)
    torch.cuda.synchronize()
    assert float(G.d_lr.item()) == 0.0
    assert torch.equal(w_before, G.st.w)
    # the schedule may run without any learning-rate buffer
    B.lamb_step(G.plan.handle, hyp, G.d_step.data_ptr(), 0)
    torch.cuda.synchronize()
    G.close()
