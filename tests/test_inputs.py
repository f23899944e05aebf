"""The synthetic inputs follow their stated recipes.

They stand in for the paper's pooled CNN features (Section 4: YFCC100M, the
Instagram-Food set, 256-dimensional PCA features clustered with K = 50), which
are not available.  Checked here, on the CPU and on small row counts of each
recipe: the sizes and element types of the five workloads, seeding, the
mixture weights (uniform, or Zipf with the largest-component shares that the
closed forms give), the drawn component frequencies, the post-ReLU zero
fraction, unit-norm rows, the noise scale around each centre, and the tag
lists (Poisson counts, Zipf vocabulary, CSR structure).
"""
import math

import numpy as np
import pytest
import torch

import hme_synth

W = hme_synth.WORKLOADS
EULER_GAMMA = 0.5772156649015329

# workload: (N, d, K, element type, Lloyd iterations)
SIZES = {
    1: (10_000, 128, 16, "f32", 10),
    2: (1_000_000, 2048, 64, "f32", 20),
    3: (4_000_000, 2048, 256, "bf16", 20),
    4: (16_000_000, 512, 1024, "f32", 10),
    5: (50_000_000, 256, 4096, "bf16", 5),
}


def _largest_share(w):
    p = hme_synth.component_weights(w)
    return float(p[0] / p.sum())


def test_workload_sizes():
    assert sorted(W) == sorted(SIZES)
    for i, (N, d, K, dt, iters) in SIZES.items():
        w = W[i]
        assert (w.N, w.d, w.K, w.dtype, w.iters) == (N, d, K, dt, iters), w.name
        assert w.comps == w.K  # one generating component per centre
        assert w.elem_bytes == (4 if dt == "f32" else 2)


@pytest.mark.parametrize("i", sorted(W))
def test_features_are_seeded_and_typed(i):
    w = W[i]
    X1, c1 = hme_synth.make_features(w, N=257)
    X2, c2 = hme_synth.make_features(w, N=257)
    assert X1.shape == (257, w.d) and X1.dtype == (torch.float32 if w.dtype == "f32" else torch.bfloat16)
    assert torch.equal(X1, X2) and torch.equal(c1, c2)
    assert int(c1.min()) >= 0 and int(c1.max()) < w.comps
    h = hme_synth.host_array(X1, w.dtype)
    if w.dtype == "bf16":  # the oracle's view: the same 16-bit patterns
        assert h.dtype == np.uint16
        assert np.array_equal(h, X1.view(torch.int16).numpy().view(np.uint16))
    else:
        assert h.dtype == np.float32 and np.array_equal(h, X1.numpy())


def test_workloads_draw_different_numbers():
    a, _ = hme_synth.make_features(W[2], N=64)
    b, _ = hme_synth.make_features(W[3], N=64)
    assert not torch.equal(a, b.float())


def test_zipf_weights_closed_forms():
    # uniform mixtures
    for i in (1, 2, 4):
        p = hme_synth.component_weights(W[i])
        assert torch.all(p == p[0])
    # Zipf(1.0) over 4096 components: the largest share is 1 / H_4096, and
    # H_n = ln n + gamma + 1 / (2n) - 1 / (12 n^2) + O(n^-4)
    n = 4096
    H = math.log(n) + EULER_GAMMA + 1 / (2 * n) - 1 / (12 * n * n)
    assert abs(_largest_share(W[5]) - 1 / H) < 1e-9
    # Zipf(1.1) over 256 components: sum_k k^-1.1 = zeta(1.1) - tail, the tail
    # by Euler-Maclaurin: int_256^inf x^-1.1 dx - 256^-1.1 / 2 + ...
    zeta_11 = 10.584448464950810  # zeta(1.1)
    tail = 10 * 256 ** -0.1 - 0.5 * 256 ** -1.1 + (1.1 / 12) * 256 ** -2.1
    assert abs(_largest_share(W[3]) - 1 / (zeta_11 - tail)) < 1e-6
    assert 0.205 < _largest_share(W[3]) < 0.209  # the largest component holds about 21% of the points


@pytest.mark.parametrize("i,N", [(3, 20_000), (5, 100_000), (2, 20_000)])
def test_drawn_component_frequencies(i, N):
    w = W[i]
    _, comp = hme_synth.make_features(w, N=N)
    p = hme_synth.component_weights(w)
    p = (p / p.sum()).numpy()
    freq = np.bincount(comp.numpy(), minlength=w.comps) / N
    sigma = np.sqrt(p * (1 - p) / N)
    assert np.all(np.abs(freq - p) <= 5 * sigma + 1e-12)


@pytest.mark.parametrize("i", [2, 3])
def test_post_relu_features_are_about_half_zeros(i):
    X, _ = hme_synth.make_features(W[i], N=2000)
    zeros = float((X == 0).float().mean())
    assert abs(zeros - hme_synth.expected_zero_fraction(W[i])) < 0.01
    assert float(X.min()) == 0.0


def test_features_without_relu_have_no_zeros():
    for i in (1, 5):
        X, _ = hme_synth.make_features(W[i], N=2000)
        assert float((X == 0).float().mean()) < 1e-3


def test_l2_normalised_rows():
    X, _ = hme_synth.make_features(W[4], N=5000)
    norms = X.double().norm(dim=1)
    assert torch.all((norms - 1).abs() < 1e-5)


def test_noise_scale_and_centre_spread():
    """Workload 1: unit noise around centres drawn with standard deviation 4."""
    w = W[1]
    X, comp = hme_synth.make_features(w, N=w.N)
    X = X.double()
    means = torch.stack([X[comp == k].mean(0) for k in range(w.comps)])
    resid = X - means[comp.long()]
    noise_var = float(resid.pow(2).mean())
    assert abs(noise_var - w.noise_std ** 2) < 0.02
    centre_var = float(means.pow(2).mean())  # the centres have mean 0
    assert abs(centre_var - w.center_std ** 2) < 0.15 * w.center_std ** 2


def test_tag_lists():
    w = W[4]
    N = 20_000
    tag_off, tags = hme_synth.make_tags(w, N=N)
    assert tag_off.dtype == torch.int64 and tags.dtype == torch.int32
    assert int(tag_off[0]) == 0 and int(tag_off[-1]) == tags.numel()
    counts = (tag_off[1:] - tag_off[:-1]).double()
    assert torch.all(counts >= 0)
    # Poisson(3): mean and variance 3
    assert abs(float(counts.mean()) - w.tag_mean) < 5 * math.sqrt(w.tag_mean / N)
    assert abs(float(counts.var()) - w.tag_mean) < 0.15
    # Zipf(1.0) over 20000 words: the most frequent tag has share 1 / H_20000
    assert int(tags.min()) >= 0 and int(tags.max()) < w.tag_vocab
    T = tags.numel()
    H = math.log(w.tag_vocab) + EULER_GAMMA + 1 / (2 * w.tag_vocab)
    share0 = float((tags == 0).double().mean())
    assert abs(share0 - 1 / H) < 5 * math.sqrt((1 / H) * (1 - 1 / H) / T)
    X1, _ = hme_synth.make_tags(w, N=N)
    assert torch.equal(X1, tag_off)  # seeded
