"""GPU test of the data-parallel (sharded) step on one GPU: two plans over
disjoint chunk ranges of one layout (ranks 0 and 1 of 2), bound to the same
state, run lamb_shard_pass1, their sum arrays are added (the all-reduce a
multi-GPU caller does), and lamb_shard_pass2 finishes the step.  The state
and the trust ratios must equal one unsharded step bit for bit (same chunk
table: same sizes, chunk size and tail)."""
import numpy as np
import pytest
import torch

from gpu_util import GpuLayout, c_hyper, f32
from paper_1904_00962_gb300 import binding as B
from paper_1904_00962_gb300 import build as build_mod
from paper_1904_00962_gb300 import workloads as W
from paper_1904_00962_gb300.state import DeviceState, LambPlan

pytestmark = pytest.mark.gpu

TAIL = 6000
SIZES = [0, 1, 3, 1023, 1024, 1025, 16383, 16384, 16385, 65539, 0, 3000,
         100003]


@pytest.fixture(scope="module", autouse=True)
def _lib(gpu):
    build_mod.build()
    B.load()
    yield
    torch.cuda.empty_cache()


def _layout(grad_dtype, copy_dtype):
    n = len(SIZES)
    return W.Layout(name="shard_gpu", names=[f"s{i}" for i in range(n)],
                    shapes=[(s,) for s in SIZES],
                    decay=[i % 2 for i in range(n)],
                    init=[("normal", 0.02)] * n,
                    grad_sigma=[10 ** (-2 - (i % 4)) for i in range(n)],
                    grad_dtype=grad_dtype, copy_dtype=copy_dtype,
                    zero_w={3}, zero_g={4},
                    hyper=W.Hyper(lr=2e-3, phi="clip", gamma_l=0.0,
                                  gamma_u=10.0))


def _state(L, with_v, t):
    st = DeviceState(L.sizes, grad_dtype=L.grad_dtype,
                     copy_dtype=L.copy_dtype, device="cuda:0", with_v=with_v)
    for k in range(L.n_tensors):
        st.upload("w", k, L.weights(k))
        st.upload("g", k, L.grad(k, t))
        m, v = L.state_warm(k)
        st.upload("m", k, m)
        if with_v:
            st.upload("v", k, v)
    return st


def _snap(st):
    out = [st.w.clone(), st.m.clone()]
    if st.v is not None:
        out.append(st.v.clone())
    if st.copy is not None:
        out.append(st.copy.view(torch.int16).clone())
    return out


@pytest.mark.parametrize("opt", ["lamb", "lars", "nlamb", "nnlamb"])
@pytest.mark.parametrize("grad_dtype,copy_dtype", [("f32", None),
                                                    ("bf16", "bf16")])
def test_two_shards_equal_one_unsharded_step_bitwise(opt, grad_dtype,
                                                     copy_dtype):
    L = _layout(grad_dtype, copy_dtype)
    lars = opt == "lars"
    h = (W.Hyper(lr=0.5, trust_coef=1e-3, weight_decay=1e-4,
                 bias_correction=False) if lars else L.hyper)
    code = {"lamb": B.LAMB_OPT_LAMB, "lars": B.LAMB_OPT_LARS,
            "nlamb": B.LAMB_OPT_NLAMB, "nnlamb": B.LAMB_OPT_NNLAMB}[opt]
    hyp = c_hyper(h, lars=lars, increment=True)
    t, psi = 5, 0.004
    dev = "cuda:0"

    def scalars():
        return (torch.full((1,), t, dtype=torch.int64, device=dev),
                torch.full((1,), f32(h.lr), dtype=torch.float32, device=dev),
                torch.full((1,), 0.6, dtype=torch.float64, device=dev))

    # one unsharded step
    su = _state(L, not lars, t)
    pu = LambPlan(su, L.decay, algorithm=B.LAMB_ALGO_TWO_PASS,
                  tail_elems=TAIL)
    d_step, d_lr, d_prod = scalars()
    if opt == "lamb":
        pu.lamb_step(hyp, d_step, d_lr)
    elif lars:
        pu.lars_step(hyp, d_step, d_lr)
    else:
        pu.nlamb_step(hyp, psi, opt == "nnlamb", d_step, d_lr, d_prod)
    want = _snap(su) + list(pu.results())
    want_t, want_prod = int(d_step.item()), float(d_prod.item())

    # two shards over one state, each with its own step scalars
    ss = _state(L, not lars, t)
    plans = [LambPlan(ss, L.decay, algorithm=B.LAMB_ALGO_TWO_PASS,
                      tail_elems=TAIL, shard_world=2, shard_rank=r)
             for r in range(2)]
    infos = [p.info() for p in plans]
    assert infos[0]["shard_chunk_begin"] == 0
    assert infos[0]["shard_chunk_end"] == infos[1]["shard_chunk_begin"]
    assert infos[1]["shard_chunk_end"] == infos[0]["n_chunks"]
    sc = [scalars() for _ in plans]
    for r in (1, 0):                                  # order does not matter
        plans[r].shard_pass1(hyp, code, *sc[r], momentum_decay=psi)
    # what an in-place all-reduce (sum) over the two ranks leaves in each
    total = plans[0].partials() + plans[1].partials()
    for p in plans:
        p.set_partials(total)
    for r in (0, 1):
        plans[r].shard_pass2(hyp, code, *sc[r], momentum_decay=psi)
    torch.cuda.synchronize()
    got = _snap(ss)
    for a, b in zip(got, want):
        assert torch.equal(a, b)
    for p in plans:
        for a, b in zip(p.results(), want[len(got):]):
            assert torch.equal(a, b)
        assert p.query() == 0
    for s in sc:
        assert int(s[0].item()) == want_t
        if opt in ("nlamb", "nnlamb"):
            assert float(s[2].item()) == want_prod
    pu.destroy()
    for p in plans:
        p.destroy()


def test_sharded_plan_rejects_the_plain_entry_points_and_grad_check():
    L = _layout("f32", None)
    st = _state(L, True, 2)
    p = LambPlan(st, L.decay, algorithm=B.LAMB_ALGO_TWO_PASS,
                 tail_elems=TAIL, shard_world=2, shard_rank=1)
    d_step = torch.ones(1, dtype=torch.int64, device="cuda:0")
    d_lr = torch.ones(1, dtype=torch.float32, device="cuda:0")
    with pytest.raises(B.LambError) as ei:
        p.lamb_step(c_hyper(L.hyper), d_step, d_lr)
    assert ei.value.status == B.LAMB_ERR_INVALID_ARG
    with pytest.raises(B.LambError) as ei:
        B.lamb_shard_pass1(p.handle, B.make_hyper(grad_norm=True),
                           B.LAMB_OPT_LAMB, 0.0, d_step.data_ptr(),
                           d_lr.data_ptr(), 0, 0)
    assert ei.value.status == B.LAMB_ERR_INVALID_ARG
    with pytest.raises(B.LambError):
        LambPlan(st, L.decay, shard_world=2, shard_rank=2)
    p.destroy()
