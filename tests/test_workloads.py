"""The seeded input generators (CPU): reproducible, with the shapes and the statistical
structure the synthetic workloads claim to stand in for.  These are input recipes, not
the method: the tests pin what the bench and the parity tests rely on."""
import math

import numpy as np
import pytest
import torch

from paper_2608_28113_gb300 import workloads as wl


def test_seeds_are_reproducible_and_distinct():
    assert wl.chunk_seed(3, "x", 0) == wl.chunk_seed(3, "x", 0)
    seeds = {wl.chunk_seed(s, st, i) for s in (0, 1, 4) for st in ("w", "a", "x") for i in range(8)}
    assert len(seeds) == 3 * 3 * 8
    assert all(0 <= v < 2 ** 63 for v in seeds)
    a = wl.weight(64, 128, 0.02, 7)
    b = wl.weight(64, 128, 0.02, 7)
    c = wl.weight(64, 128, 0.02, 8)
    assert a.dtype == torch.bfloat16 and a.shape == (64, 128)
    assert torch.equal(a, b) and not torch.equal(a, c)


def test_weight_distribution_and_outliers():
    """Student-t(4) * sigma: excess kurtosis well above a Gaussian's, round(0.1 % m n)
    outliers x20, and the scale sigma on the bulk."""
    m, n, sigma = 512, 1024, 0.02
    w = wl.weight(m, n, sigma, 3).float()
    base = wl.weight(m, n, sigma, 3, outlier_frac=0.0).float()
    changed = (w != base).sum().item()
    k = round(1e-3 * m * n)
    # an outlier can only go unnoticed if its entry is zero in bf16
    assert k - 2 <= changed <= k
    ratio = (w[w != base] / base[w != base])
    assert torch.allclose(ratio, torch.full_like(ratio, 20.0), rtol=1e-2)
    x = base.flatten().double()
    # Student-t(4): variance nu / (nu - 2) = 2 in units of sigma^2
    assert abs(x.var().item() / (2 * sigma ** 2) - 1) < 0.15
    kurt = ((x - x.mean()) ** 4).mean() / x.var() ** 2 - 3
    assert kurt > 2.0


def test_channel_magnitudes_and_activations():
    """a_c ~ LogNormal(0, sigma_a) with `outliers` channels x mult; X = N(0, 1) a_c per
    channel, i.i.d. tokens, so the column mean square of X tracks a_c^2."""
    n = 2048
    a = wl.channel_magnitudes(n, 1.0, 8, 50.0, 11)
    base = wl.channel_magnitudes(n, 1.0, 0, 50.0, 11)
    big = torch.nonzero(a != base).flatten()
    assert big.numel() == 8 and torch.allclose(a[big] / base[big], torch.full((8,), 50.0))
    la = torch.log(base.double())
    assert abs(la.mean().item()) < 0.1 and abs(la.std().item() - 1.0) < 0.1
    x = wl.activation_chunk(4096, a, 11, 0)
    assert x.dtype == torch.bfloat16 and x.shape == (4096, n)
    ms = (x.double() ** 2).mean(0)
    rel = ms / (a.double() ** 2)
    # the mean of 4096 chi-square(1) draws: within 5 standard errors of 1
    assert (rel - 1).abs().max().item() < 5 * math.sqrt(2 / 4096) + 0.01
    # chunks of one stream differ, and the same index reproduces
    assert torch.equal(x, wl.activation_chunk(4096, a, 11, 0))
    assert not torch.equal(x[:64], wl.activation_chunk(64, a, 11, 1))


def test_activation_chunk_writes_into_a_view():
    a = wl.channel_magnitudes(256, 1.5, 4, 100.0, 2)
    out = torch.zeros(300, 256, dtype=torch.bfloat16)
    wl.activation_chunk(128, a, 2, 3, out=out[100:228])
    assert torch.equal(out[100:228], wl.activation_chunk(128, a, 2, 3))
    assert out[:100].abs().sum().item() == 0 and out[228:].abs().sum().item() == 0


def test_bf16_bits_views_the_bit_patterns():
    t = torch.tensor([1.0, -2.0, 0.5, 0.0, -0.0], dtype=torch.bfloat16)
    b = wl.bf16_bits(t)
    assert b.dtype == np.uint16
    assert b.tolist() == [0x3F80, 0xC000, 0x3F00, 0x0000, 0x8000]
    with pytest.raises(TypeError):
        wl.bf16_bits(torch.zeros(2))


@pytest.mark.parametrize("name", sorted(wl.WORKLOADS))
def test_workload_shapes_are_consistent(name):
    """Every matrix's width is a whole number of 16-element groups and of its input
    space's streamed chunk recipe; matrices sharing an input space share its width."""
    W = wl.WORKLOADS[name]
    spaces = dict(W.input_spaces())
    for L in W.layers:
        assert L.in_features % 16 == 0 and L.out_features > 0
        assert spaces[L.input_space] == L.in_features
        assert W.chunk_tokens[L.in_features] > 0
    assert all(k >= 0 for k in W.window)
    assert W.layer_seed(0) == (W.seed if W.n_layers == 1 else W.seed * 1000)
