"""Pins of the PCA oracle (Section 4.2: projection onto the leading principal
directions before the K-means) against facts that do not come from the oracle
itself: a data set built with a known covariance, the 2 x 2 closed form,
invariants of an eigendecomposition and of the projection, an independent SVD
route, power iteration on a tiny case and the Ky Fan maximum principle."""
import numpy as np
import pytest

from oracle import pca


def _orthogonal(d, seed):
    """A seeded orthogonal matrix (Householder QR of a Gaussian matrix)."""
    q, r = np.linalg.qr(np.random.default_rng(seed).standard_normal((d, d)))
    return q * np.sign(np.diag(r))


def _known_spectrum(d, lam, mu, seed):
    """2d rows mu +- sqrt(d lam_j) q_j: column mean mu exactly, covariance
    (1/N) sum = Q diag(lam) Q^T with N = 2d."""
    Q = _orthogonal(d, seed)
    rows = []
    for j in range(d):
        a = np.sqrt(d * lam[j]) * Q[:, j]
        rows += [mu + a, mu - a]
    return np.array(rows), Q


def test_known_spectrum_and_directions():
    d = 12
    lam = np.array([9.0, 7.5, 6.0, 4.0, 3.0, 2.5, 2.0, 1.5, 1.0, 0.5, 0.25, 0.125])
    mu = np.linspace(-3.0, 5.0, d)  # a non-zero mean: centring must happen
    X, Q = _known_spectrum(d, lam, mu, seed=3)
    m, W, l, C = pca.fit(X, 5)
    assert np.allclose(m, mu, rtol=0, atol=1e-12)
    assert np.allclose(l, lam, rtol=1e-12, atol=1e-12)  # decreasing, normalised by N
    assert np.allclose(C, Q @ np.diag(lam) @ Q.T, atol=1e-12)
    ref = pca.canonical_signs(Q[:, :5].T)
    assert np.allclose(W, ref, atol=1e-10)
    for k in range(5):  # the sign rule: the largest-magnitude entry is positive
        assert W[k, np.argmax(np.abs(W[k]))] > 0


def test_projection_of_the_known_spectrum_rows():
    """Row mu +- sqrt(d lam_j) q_j projects to +- sqrt(d lam_j) s_j e_j on the
    r leading components (s_j the component's sign) and to 0 for j >= r."""
    d, r = 10, 4
    lam = np.array([8.0, 6.0, 5.0, 3.0, 2.0, 1.5, 1.0, 0.6, 0.3, 0.1])
    mu = np.linspace(2.0, -1.0, d)
    X, Q = _known_spectrum(d, lam, mu, seed=17)
    m, W, _, _ = pca.fit(X, r)
    Z = pca.transform(X, m, W)
    signs = np.sign(np.sum(W * Q[:, :r].T, axis=1))  # W[k] = s_k q_k
    for j in range(d):
        want = np.zeros(r)
        if j < r:
            want[j] = signs[j] * np.sqrt(d * lam[j])
        assert np.allclose(Z[2 * j], want, atol=1e-9)
        assert np.allclose(Z[2 * j + 1], -want, atol=1e-9)


def test_two_by_two_closed_form():
    rng = np.random.default_rng(7)
    X = rng.standard_normal((500, 2)) @ np.array([[2.0, 0.7], [0.0, 0.9]]) + np.array([4.0, -1.0])
    _, W, l, C = pca.fit(X, 2)
    a, b, c = C[0, 0], C[0, 1], C[1, 1]
    h = np.hypot((a - c) / 2, b)
    assert np.allclose(l, [(a + c) / 2 + h, (a + c) / 2 - h], rtol=1e-12)
    theta = 0.5 * np.arctan2(2 * b, a - c)  # direction of the larger eigenvalue
    v = pca.canonical_signs(np.array([[np.cos(theta), np.sin(theta)]]))[0]
    assert np.allclose(W[0], v, atol=1e-12)


def test_eigendecomposition_and_projection_invariants():
    rng = np.random.default_rng(11)
    N, d, r = 3000, 40, 9
    X = np.maximum(rng.standard_normal((N, d)) + 2 * rng.standard_normal((6, d))[rng.integers(0, 6, N)], 0)
    X = X.astype(np.float32)
    mu, W, lam, C = pca.fit(X, r)
    assert np.allclose(W @ W.T, np.eye(r), atol=1e-12)
    assert np.allclose(C @ W.T, W.T * lam[:r], atol=1e-10 * lam[0])
    Y = X.astype(np.float64) - mu
    assert np.isclose(lam.sum(), np.trace(C), rtol=1e-12)
    assert np.isclose(np.trace(C), np.mean(np.sum(Y * Y, axis=1)), rtol=1e-12)  # total variance
    Z = pca.transform(X, mu, W)
    assert np.allclose(Z.mean(axis=0), 0, atol=1e-10 * np.sqrt(lam[0]))
    assert np.allclose(Z.T @ Z / N, np.diag(lam[:r]), atol=1e-10 * lam[0])  # uncorrelated, variances lam
    assert np.all(np.diff(lam) <= 0)


def test_matches_the_svd_route():
    """The right singular vectors of the centred data, by LAPACK's SVD (no
    covariance formed), give the same directions and s^2 / N the same
    variances."""
    rng = np.random.default_rng(5)
    N, d, r = 800, 24, 6
    X = (rng.standard_normal((N, d)) * np.linspace(3.0, 0.2, d)) @ _orthogonal(d, 2) + 1.5
    mu, W, lam, _ = pca.fit(X, r)
    Y = X - X.mean(axis=0)
    _, s, Vt = np.linalg.svd(Y, full_matrices=False)
    assert np.allclose(lam, s ** 2 / N, rtol=1e-10)
    assert np.allclose(W, pca.canonical_signs(Vt[:r]), atol=1e-8)


def test_matches_scikit_learn():
    sk = pytest.importorskip("sklearn.decomposition")
    rng = np.random.default_rng(9)
    N, d, r = 600, 16, 5
    X = (rng.standard_normal((N, d)) * np.linspace(2.0, 0.3, d)) @ _orthogonal(d, 4) - 0.7
    mu, W, lam, _ = pca.fit(X, r)
    ref = sk.PCA(n_components=r, svd_solver="full").fit(X)
    assert np.allclose(mu, ref.mean_, atol=1e-12)
    assert np.allclose(lam[:r], ref.explained_variance_ * (N - 1) / N, rtol=1e-10)  # it divides by N - 1
    assert np.allclose(W, pca.canonical_signs(ref.components_), atol=1e-8)
    assert np.allclose(pca.transform(X, mu, W), ref.transform(X) * np.sign(np.sum(W * ref.components_, 1)),
                       atol=1e-8)


def test_power_iteration_on_a_tiny_case():
    X = np.array([[1.0, 2.0, 0.5], [2.0, 3.5, 1.0], [0.0, -1.0, 0.2], [3.0, 4.0, 2.5], [1.5, 0.5, -0.5]])
    mu, C = pca.covariance(X)
    v = np.ones(3)
    for _ in range(500):
        v = C @ v
        v /= np.linalg.norm(v)
    _, W, lam, _ = pca.fit(X, 1)
    assert np.allclose(W[0], pca.canonical_signs(v[None])[0], atol=1e-12)
    assert np.isclose(lam[0], v @ C @ v, rtol=1e-12)


def test_leading_components_maximise_captured_variance():
    """Ky Fan: no r-dimensional orthonormal basis captures more variance than
    the r leading components."""
    rng = np.random.default_rng(13)
    N, d, r = 400, 10, 3
    X = rng.standard_normal((N, d)) * np.linspace(3.0, 0.5, d)
    _, W, lam, C = pca.fit(X, r)
    best = np.trace(W @ C @ W.T)
    assert np.isclose(best, lam[:r].sum(), rtol=1e-12)
    for s in range(200):
        B = _orthogonal(d, 100 + s)[:r]
        assert np.trace(B @ C @ B.T) <= best * (1 + 1e-12)
