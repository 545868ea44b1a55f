"""CPU tests of the data-parallel (sharded) step's host logic, world size 2
and 3 over gloo.  Each rank takes its chunk range from the library's host
planner (lamb_layout_shard over lamb_layout_chunks), forms the per-chunk
sums of w^2 and u^2 of its elements with the fp64 oracle's element-wise part
(Alg. 2 moment and ratio lines; Alg. 1 momentum for LARS), all-reduces them
like the caller of lamb_shard_pass1 does, forms the trust ratios from the
reduced sums, and updates its elements.  Every rank's slice must equal the
unsharded oracle step, and the ranges must cover every chunk once.  The
kernels of the same exchange run in the GPU test (test_shard_gpu.py)."""
import math
import os
import socket
import sys

import numpy as np
import pytest

from conftest import ROOT

EDGE = [0, 1, 3, 1023, 1024, 1025, 16383, 16384, 16385, 65539, 0, 3000,
        100003]


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _layout(name):
    from paper_1904_00962_gb300 import workloads as W
    if name == "mlp":
        return W.mlp_layout()
    n = len(EDGE)
    return W.Layout(name="shard_edge", names=[f"e{i}" for i in range(n)],
                    shapes=[(s,) for s in EDGE],
                    decay=[i % 2 for i in range(n)],
                    init=[("normal", 0.02)] * n,
                    grad_sigma=[10 ** (-2 - (i % 4)) for i in range(n)],
                    zero_w={3}, zero_g={4},
                    hyper=W.Hyper(lr=2e-3, phi="clip", gamma_l=0.0,
                                  gamma_u=10.0))


def _worker(rank, world, port, name, lars, q):
    import torch
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    sys.path.insert(0, ROOT)
    from oracle import lamb_oracle as O
    from paper_1904_00962_gb300 import binding as B
    try:
        L = _layout(name)
        h = L.hyper
        chunk, tail = 4096, 6000
        t_of, off, ln = B.lamb_layout_chunks(L.sizes, chunk, tail)
        cb, ce = B.lamb_layout_shard(L.sizes, world, rank, chunk, tail)
        t, lr = 3, 2e-3 if not lars else 0.5
        kw = dict(beta1=h.beta1, weight_decay=h.weight_decay if not lars
                  else 1e-4)
        parts = torch.zeros(len(t_of), 2, dtype=torch.float64)
        dirs = {}
        for c in range(cb, ce):
            k, a, n = int(t_of[c]), int(off[c]), int(ln[c])
            w = L.weights(k)[a:a + n]
            g = L.grad(k, t)[a:a + n]
            m, v = (x[a:a + n] for x in L.state_warm(k))
            if lars:
                u = O.lars_momentum(w, g, m, decay=bool(L.decay[k]), **kw)
                mv = (u, None)
            else:
                m_t, v_t, u = O.lamb_direction(
                    w, g, m, v, t=t, beta2=h.beta2, eps=h.eps,
                    decay=bool(L.decay[k]), **kw)
                mv = (m_t, v_t)
            w64 = O.to_f64(w)
            parts[c, 0] = math.fsum((w64 * w64).tolist())
            parts[c, 1] = math.fsum((u * u).tolist())
            dirs[c] = (w64, u, mv)
        dist.all_reduce(parts)          # one non-zero contributor per entry
        # every chunk owned once: the ranges tile the table
        rng = torch.tensor([cb, ce], dtype=torch.int64)
        allr = [torch.zeros(2, dtype=torch.int64) for _ in range(world)]
        dist.all_gather(allr, rng)
        worst = 0.0
        for c in range(cb, ce):
            k, a, n = int(t_of[c]), int(off[c]), int(ln[c])
            sel = np.flatnonzero(t_of == k)
            sw = math.fsum(parts[sel, 0].tolist())
            su = math.fsum(parts[sel, 1].tolist())
            wn, un = math.sqrt(sw), math.sqrt(su)
            coef = 1e-3 if lars else 1.0
            rho = 1.0 if (wn == 0.0 or un == 0.0) else \
                coef * O.phi(wn, h.phi if not lars else "identity",
                             h.gamma_l, h.gamma_u) / un
            w64, u, (m_t, v_t) = dirs[c]
            w_new = w64 - lr * rho * u
            # the unsharded oracle step of the whole tensor, this slice
            wf, gf = L.weights(k), L.grad(k, t)
            mf, vf = L.state_warm(k)
            if lars:
                ref = O.lars_tensor(wf, gf, mf, lr=lr, decay=bool(L.decay[k]),
                                    trust_coef=1e-3, **kw)
            else:
                ref = O.lamb_tensor(wf, gf, mf, vf, t=t, lr=lr,
                                    decay=bool(L.decay[k]), beta2=h.beta2,
                                    eps=h.eps, phi_kind=h.phi,
                                    gamma_l=h.gamma_l, gamma_u=h.gamma_u,
                                    **kw)
                np.testing.assert_array_equal(v_t, ref.v[a:a + n])
            np.testing.assert_array_equal(m_t, ref.m[a:a + n])
            assert abs(rho - ref.ratio) <= 1e-12 * abs(ref.ratio), (k, rho)
            scale = np.maximum(np.abs(ref.w[a:a + n]), np.abs(w64))
            err = np.abs(w_new - ref.w[a:a + n])
            if err.size:
                worst = max(worst, float(np.max(err / np.where(
                    scale > 0, scale, 1.0))))
        q.put((rank, [tuple(int(x) for x in r) for r in allr], worst,
               len(t_of), None))
    except Exception as e:   # report, do not hang the other rank
        q.put((rank, None, None, None, repr(e)))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
@pytest.mark.parametrize("name,lars", [("mlp", False), ("edge", False),
                                       ("edge", True)])
def test_sharded_step_host_logic_matches_unsharded_oracle(world, name, lars):
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, name, lars, q))
             for r in range(world)]
    for p in procs:
        p.start()
    out = {}
    for _ in procs:
        rank, ranges, worst, n_chunks, err = q.get(timeout=300)
        assert err is None, f"rank {rank}: {err}"
        out[rank] = (ranges, worst, n_chunks)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    ranges = out[0][0]
    n_chunks = out[0][2]
    assert ranges[0][0] == 0 and ranges[-1][1] == n_chunks
    for a, b in zip(ranges, ranges[1:]):
        assert a[1] == b[0]                  # contiguous, disjoint, complete
    for rank, (_, worst, _) in out.items():
        assert worst <= 1e-13, (rank, worst)   # fp64 sum order only


def test_shard_ranges_split_elements_evenly(tmp_path):
    sys.path.insert(0, ROOT)
    from paper_1904_00962_gb300 import binding as B
    from paper_1904_00962_gb300 import build as build_mod
    from paper_1904_00962_gb300.workloads import bert_large_layout
    build_mod.build()
    B.load()
    L = bert_large_layout()
    t_of, off, ln = B.lamb_layout_chunks(L.sizes, 16384, 0)
    starts = np.concatenate([[0], np.cumsum(ln)[:-1]])
    for world in (1, 2, 8, 64):
        prev_end = 0
        for r in range(world):
            cb, ce = B.lamb_layout_shard(L.sizes, world, r, 16384, 0)
            assert cb == prev_end
            prev_end = ce
            # the range starts at the first chunk at or past its share
            target = L.n_params * r // world
            assert cb == int(np.searchsorted(starts, target, side="left"))
            owned = int(ln[cb:ce].sum())
            assert abs(owned - L.n_params / world) <= 2 * 16384 * 1.0
        assert prev_end == len(t_of)
    with pytest.raises(B.LambError):
        B.lamb_layout_shard(L.sizes, 2, 2)
