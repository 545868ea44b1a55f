"""CPU tests of the seeded synthetic layouts (architecture counts, masks,
seeding, value recipes)."""
import math

import numpy as np
import pytest

from paper_1904_00962_gb300 import workloads as W


@pytest.mark.parametrize("name,tensors,params,masked", [
    ("mlp", 4, 2410, 2),
    ("bert_base", 199, 109482240, 123),
    ("bert_large", 391, 335141888, 243),
    ("resnet50", 161, 25557032, 107),
])
def test_layout_counts(name, tensors, params, masked):
    L = W.get_layout(name)
    assert L.n_tensors == tensors
    assert L.n_params == params
    assert L.n_tensors - sum(L.decay) == masked


def test_bert_masks_biases_and_layernorm_only():
    L = W.bert_base_layout()
    for n, d in zip(L.names, L.decay):
        assert d == (0 if (n.endswith(".bias") or ".ln." in n or "_ln." in n)
                     else 1), n


def test_resnet50_structure():
    L = W.resnet50_layout()
    convs = [s for s in L.shapes if len(s) == 4]
    assert len(convs) == 53
    assert sum(1 for n in L.names if ".gamma" in n or ".beta" in n) == 106
    assert L.shapes[-2] == (1000, 2048) and L.decay[-1] == 0
    assert L.lars_hyper.trust_coef == 1e-3


def test_ragged_layout_recipe():
    L = W.ragged_layout()
    s = np.array(L.sizes)
    assert L.n_tensors == 10000
    assert s.min() >= 1 and s.max() <= 4194304
    assert len(L.zero_w) == 100 and len(L.zero_g) == 100
    assert not (L.zero_w & L.zero_g)
    frac_masked = 1 - sum(L.decay) / 10000
    assert 0.27 < frac_masked < 0.33
    # log-uniform sizes: the median sits near sqrt(4194304) = 2048
    assert 1000 < np.median(s) < 4200
    # expected total ~ n * max / ln(max) (the stated distribution)
    expect = 10000 * 4194304 / math.log(4194304)
    assert 0.85 * expect < L.n_params < 1.15 * expect


def test_seeding_is_per_tensor_and_reproducible():
    L = W.bert_base_layout()
    a = L.grad(3, 2)
    b = W.bert_base_layout().grad(3, 2)
    np.testing.assert_array_equal(a, b)
    assert not np.array_equal(L.grad(3, 1), a)
    assert not np.array_equal(L.grad(4, 2)[:100], L.grad(3, 2)[:100])


def test_bf16_grads_are_truncated_float32_draws():
    L = W.bert_layout(1, 64, 128, vocab=50, positions=8, name="tiny",
                      grad_dtype="bf16")
    Lf = W.bert_layout(1, 64, 128, vocab=50, positions=8, name="tiny")
    bits = L.grad(0, 1)
    f = Lf.grad(0, 1)
    assert bits.dtype == np.uint16
    np.testing.assert_array_equal(bits, (f.view(np.uint32) >> 16).astype(np.uint16))


def test_init_recipes():
    L = W.bert_base_layout()
    k_gamma = L.names.index("layer0.attn_ln.gamma")
    k_bias = L.names.index("layer0.q.bias")
    assert np.all(L.weights(k_gamma) == 1.0)
    assert np.all(L.weights(k_bias) == 0.0)
    w = L.weights(L.names.index("layer0.q.weight"))
    assert abs(float(np.std(w)) - 0.02) < 0.001
    sig = np.array(L.grad_sigma)
    assert sig.min() >= 1e-5 and sig.max() <= 1e-2
    R = W.ragged_layout(200)
    for k in R.zero_w:
        assert not R.weights(k).any()
    for k in R.zero_g:
        assert not R.grad(k, 1).any()
