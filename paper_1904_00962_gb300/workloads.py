"""Seeded synthetic parameter layouts and input values.

This module only builds *inputs*: tensor shapes shaped like the paper's
workloads (BERT-base/large of Section 4.1, ResNet-50 of Section 4.2, a small
MLP and a ragged stress layout), the per-tensor weight-decay mask, and seeded
random weights, gradients and optimizer state.  It contains none of the
optimizer's arithmetic; both the CUDA path and the fp64 oracle read the same
arrays from here.

Seeding: every array is drawn from NumPy's PCG64 with a SeedSequence built
from (layout seed, a hash of the layout name, the kind of array, the step,
the tensor index), so any single tensor can be regenerated on its own.
bfloat16 gradients are produced by truncating float32 draws to their top 16
bits (an input-generation choice; it is not the rounding used by the method).
"""
from __future__ import annotations

import math
import zlib
from dataclasses import dataclass, field

import numpy as np

__all__ = ["Layout", "Hyper", "LAYOUTS", "get_layout", "mlp_layout",
           "bert_layout", "resnet50_layout", "ragged_layout"]

_KIND_IDS = {"w": 1, "g": 2, "m": 3, "v": 4, "sigma": 5, "layout": 6}


@dataclass
class Hyper:
    """Hyperparameters of one workload (Section 4 and the appendix)."""
    lr: float = 1e-3
    beta1: float = 0.9
    beta2: float = 0.999
    eps: float = 1e-6
    weight_decay: float = 0.01
    phi: str = "identity"          # "identity" | "clip"
    gamma_l: float = 0.0
    gamma_u: float = math.inf
    trust_coef: float = 1.0        # LARS only
    bias_correction: bool = True
    start_step: int = 1            # t of the first step
    warm_steps: int = 0            # steps run before the measured one
    measured_step: int | None = None   # t forced for the measured step


@dataclass
class Layout:
    name: str
    names: list
    shapes: list
    decay: list                    # 1 = weight decay applies
    init: list                     # ("normal", std) | ("const", c)
    grad_sigma: list               # per-tensor gradient std
    grad_dtype: str = "f32"        # "f32" | "bf16"
    copy_dtype: str | None = None  # None | "bf16"
    seed: int = 1234
    zero_w: set = field(default_factory=set)   # tensors with w == 0
    zero_g: set = field(default_factory=set)   # tensors with g == 0
    hyper: Hyper = field(default_factory=Hyper)
    lars_hyper: Hyper | None = None

    @property
    def sizes(self) -> list:
        return [int(np.prod(s, dtype=np.int64)) for s in self.shapes]

    @property
    def n_tensors(self) -> int:
        return len(self.shapes)

    @property
    def n_params(self) -> int:
        return int(sum(self.sizes))

    # -- seeded values ----------------------------------------------------
    def _rng(self, kind: str, step: int, k: int) -> np.random.Generator:
        ss = np.random.SeedSequence(
            [self.seed, zlib.crc32(self.name.encode()), _KIND_IDS[kind],
             int(step), int(k)])
        return np.random.Generator(np.random.PCG64(ss))

    def weights(self, k: int) -> np.ndarray:
        n = self.sizes[k]
        if k in self.zero_w:
            return np.zeros(n, dtype=np.float32)
        kind, val = self.init[k]
        if kind == "const":
            return np.full(n, val, dtype=np.float32)
        rng = self._rng("w", 0, k)
        return (rng.standard_normal(n, dtype=np.float32) * np.float32(val))

    def grad(self, k: int, step: int) -> np.ndarray:
        """float32 array, or uint16 bfloat16 bit patterns for bf16 layouts."""
        n = self.sizes[k]
        if k in self.zero_g:
            g = np.zeros(n, dtype=np.float32)
        else:
            rng = self._rng("g", step, k)
            g = rng.standard_normal(n, dtype=np.float32) * np.float32(
                self.grad_sigma[k])
        if self.grad_dtype == "bf16":
            # top half of each little-endian float32 word
            return np.ascontiguousarray(g.view(np.uint16)[1::2])
        return g

    def state_zero(self, k: int):
        n = self.sizes[k]
        return np.zeros(n, dtype=np.float32), np.zeros(n, dtype=np.float32)

    def state_warm(self, k: int):
        """Synthetic 'after a few steps' moments: m ~ N(0, 0.3 sigma_k),
        v = sigma_k^2 * U(5e-4, 3e-3) (positive), as float32."""
        n = self.sizes[k]
        s = float(self.grad_sigma[k])
        rng = self._rng("m", 0, k)
        m = rng.standard_normal(n, dtype=np.float32) * np.float32(0.3 * s)
        rng = self._rng("v", 0, k)
        v = rng.uniform(5e-4, 3e-3, n).astype(np.float32) * np.float32(s * s)
        return m, v


def _loguniform_sigmas(name: str, n: int, lo: float, hi: float, seed: int):
    ss = np.random.SeedSequence([seed, zlib.crc32(name.encode()),
                                 _KIND_IDS["sigma"]])
    rng = np.random.Generator(np.random.PCG64(ss))
    return list(np.exp(rng.uniform(math.log(lo), math.log(hi), n)))


# ---------------------------------------------------------------------------
# Layout builders
# ---------------------------------------------------------------------------

def mlp_layout() -> Layout:
    """Tiny MLP: [64,32],[32],[32,10],[10] = 2,410 parameters; biases are
    masked from decay; w ~ N(0, 0.02), g ~ N(0, 0.01); 10 chained steps."""
    shapes = [(64, 32), (32,), (32, 10), (10,)]
    names = ["fc1.weight", "fc1.bias", "fc2.weight", "fc2.bias"]
    return Layout(
        name="mlp", names=names, shapes=shapes, decay=[1, 0, 1, 0],
        init=[("normal", 0.02)] * 4, grad_sigma=[0.01] * 4,
        hyper=Hyper(lr=1e-3, phi="identity", start_step=1, warm_steps=0))


def bert_layout(layers: int, hidden: int, ffn: int, *, vocab: int = 30522,
                positions: int = 512, types: int = 2, name: str = "bert",
                grad_dtype: str = "f32", copy_dtype: str | None = None,
                measured_step: int | None = None) -> Layout:
    """BERT encoder parameter list (embeddings, `layers` transformer blocks
    of 16 tensors each, pooler).  Biases and LayerNorm gamma/beta are masked
    from decay.  Matrices ~ N(0, 0.02), LayerNorm gamma = 1, beta = 0,
    biases 0.  Per-tensor gradient std is log-uniform in [1e-5, 1e-2]."""
    names, shapes, decay, init = [], [], [], []

    def add(n, s, d, i):
        names.append(n); shapes.append(tuple(s)); decay.append(d); init.append(i)

    H, F = hidden, ffn
    add("emb.word", (vocab, H), 1, ("normal", 0.02))
    add("emb.pos", (positions, H), 1, ("normal", 0.02))
    add("emb.type", (types, H), 1, ("normal", 0.02))
    add("emb.ln.gamma", (H,), 0, ("const", 1.0))
    add("emb.ln.beta", (H,), 0, ("const", 0.0))
    for l in range(layers):
        p = f"layer{l}."
        for proj in ("q", "k", "v", "o"):
            add(p + proj + ".weight", (H, H), 1, ("normal", 0.02))
            add(p + proj + ".bias", (H,), 0, ("const", 0.0))
        add(p + "attn_ln.gamma", (H,), 0, ("const", 1.0))
        add(p + "attn_ln.beta", (H,), 0, ("const", 0.0))
        add(p + "ffn_in.weight", (F, H), 1, ("normal", 0.02))
        add(p + "ffn_in.bias", (F,), 0, ("const", 0.0))
        add(p + "ffn_out.weight", (H, F), 1, ("normal", 0.02))
        add(p + "ffn_out.bias", (H,), 0, ("const", 0.0))
        add(p + "out_ln.gamma", (H,), 0, ("const", 1.0))
        add(p + "out_ln.beta", (H,), 0, ("const", 0.0))
    add("pooler.weight", (H, H), 1, ("normal", 0.02))
    add("pooler.bias", (H,), 0, ("const", 0.0))
    sig = _loguniform_sigmas(name, len(shapes), 1e-5, 1e-2, 1234)
    hyper = Hyper(lr=2e-3, phi="clip", gamma_l=0.0, gamma_u=10.0,
                  start_step=1, warm_steps=3, measured_step=measured_step)
    return Layout(name=name, names=names, shapes=shapes, decay=decay,
                  init=init, grad_sigma=sig, grad_dtype=grad_dtype,
                  copy_dtype=copy_dtype, hyper=hyper)


def bert_base_layout() -> Layout:
    """BERT-base: 12 layers, hidden 768, FFN 3072: 199 tensors,
    109,482,240 parameters, 123 masked."""
    return bert_layout(12, 768, 3072, name="bert_base")


def bert_large_layout() -> Layout:
    """BERT-large: 24 layers, hidden 1024, FFN 4096: 391 tensors,
    335,141,888 parameters, 243 masked.  bf16 gradients, fp32 master
    weights and moments, a bf16 weight copy written every step; measured at
    t = 1000 after three warm-up steps."""
    return bert_layout(24, 1024, 4096, name="bert_large", grad_dtype="bf16",
                       copy_dtype="bf16", measured_step=1000)


def resnet50_layout() -> Layout:
    """ResNet-50 (bottleneck stages [3,4,6,3], widths [64,128,256,512] x4):
    53 conv kernels [out,in,k,k], 106 BatchNorm gamma/beta, FC 2048x1000 and
    its bias = 161 tensors, 25,557,032 parameters.  BN gamma/beta and the FC
    bias are masked.  Convs He-normal, BN gamma 1 / beta 0, FC N(0, 0.01),
    g ~ N(0, 1e-3).  LAMB uses the paper's 16K-batch ResNet learning rate
    4/(2^0.5*100); LARS uses momentum 0.9 and trust coefficient 0.001."""
    names, shapes, decay, init = [], [], [], []

    def add(n, s, d, i):
        names.append(n); shapes.append(tuple(s)); decay.append(d); init.append(i)

    def conv(n, o, i, k):
        add(n, (o, i, k, k), 1, ("normal", math.sqrt(2.0 / (i * k * k))))

    def bn(n, c):
        add(n + ".gamma", (c,), 0, ("const", 1.0))
        add(n + ".beta", (c,), 0, ("const", 0.0))

    conv("conv1", 64, 3, 7)
    bn("bn1", 64)
    cin = 64
    for s, (blocks, width) in enumerate(zip([3, 4, 6, 3], [64, 128, 256, 512])):
        for b in range(blocks):
            p = f"layer{s + 1}.{b}."
            conv(p + "conv1", width, cin, 1); bn(p + "bn1", width)
            conv(p + "conv2", width, width, 3); bn(p + "bn2", width)
            conv(p + "conv3", 4 * width, width, 1); bn(p + "bn3", 4 * width)
            if b == 0:
                conv(p + "downsample", 4 * width, cin, 1)
                bn(p + "downsample_bn", 4 * width)
            cin = 4 * width
    add("fc.weight", (1000, 2048), 1, ("normal", 0.01))
    add("fc.bias", (1000,), 0, ("const", 0.0))
    hyper = Hyper(lr=4.0 / (2 ** 0.5 * 100), phi="clip", gamma_l=0.0,
                  gamma_u=10.0, start_step=1, warm_steps=3)
    lars = Hyper(lr=10.0, beta1=0.9, weight_decay=1e-4, phi="identity",
                 trust_coef=1e-3, bias_correction=False, start_step=1,
                 warm_steps=3)
    return Layout(name="resnet50", names=names, shapes=shapes, decay=decay,
                  init=init, grad_sigma=[1e-3] * len(shapes), hyper=hyper,
                  lars_hyper=lars)


def ragged_layout(n: int = 10000, max_size: int = 4194304,
                  seed: int = 4321) -> Layout:
    """Ragged stress layout: `n` tensors with sizes floor(exp(U(0, ln
    max_size))) >= 1, 30% masked from decay, 1% all-zero weights and 1%
    all-zero gradients (disjoint random picks).  w ~ N(0, 0.02),
    g ~ N(0, 1e-3), m = v = 0, t = 1."""
    ss = np.random.SeedSequence([seed, zlib.crc32(b"ragged"),
                                 _KIND_IDS["layout"], n])
    rng = np.random.Generator(np.random.PCG64(ss))
    sizes = np.floor(np.exp(rng.uniform(0.0, math.log(max_size), n)))
    sizes = np.maximum(sizes.astype(np.int64), 1)
    decay = (rng.uniform(0, 1, n) >= 0.3).astype(int).tolist()
    picks = rng.permutation(n)
    n1 = max(1, n // 100)
    zero_w = set(int(i) for i in picks[:n1])
    zero_g = set(int(i) for i in picks[n1:2 * n1])
    name = "ragged" if n == 10000 else f"ragged{n}"
    hyper = Hyper(lr=2e-3, phi="clip", gamma_l=0.0, gamma_u=10.0,
                  start_step=1, warm_steps=0)
    return Layout(name=name, names=[f"t{i}" for i in range(n)],
                  shapes=[(int(s),) for s in sizes], decay=decay,
                  init=[("normal", 0.02)] * n, grad_sigma=[1e-3] * n,
                  zero_w=zero_w, zero_g=zero_g, seed=seed, hyper=hyper)


LAYOUTS = {
    "mlp": mlp_layout,
    "bert_base": bert_base_layout,
    "bert_large": bert_large_layout,
    "resnet50": resnet50_layout,
    "ragged": ragged_layout,
}


def get_layout(name: str) -> Layout:
    if name.startswith("ragged") and name != "ragged":
        return ragged_layout(int(name[len("ragged"):]))
    return LAYOUTS[name]()
