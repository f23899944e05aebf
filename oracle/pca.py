"""fp64 CPU oracle for the PCA projection that precedes the gater's K-means
(arXiv 1704.06363, Section 4.2, "Model and training details": before the
clustering, the gater features Z = T^{L-1}(X) are projected onto their first
256 principal directions).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
module; the product path never imports it and it imports nothing of the
product path.

The paper names the method and the dimension only.  Readings taken here:
  * centred: principal directions of the covariance about the column mean;
  * the covariance is normalised by N (the variance of the data), so the
    reported variances are the eigenvalues of (1/N) sum_i (x_i - mu)(x_i - mu)^T;
  * unwhitened: z = W (x - mu) with orthonormal component rows, no 1/sqrt(lambda);
  * components ordered by decreasing variance; each component's sign is chosen
    so that its entry of largest magnitude is positive (the lowest index among
    entries of equal magnitude).
Steps, in order: mean (fp64), covariance as a product of the centred fp64 rows
(a library matrix product), the symmetric eigendecomposition
(numpy.linalg.eigh, a library routine), ordering, sign rule, projection.
Features are float32 arrays; every step is fp64.
"""
from __future__ import annotations

import numpy as np


def mean(X) -> np.ndarray:
    """Column mean mu_j = (1/N) sum_i x_ij, fp64."""
    X = np.asarray(X)
    return X.astype(np.float64).mean(axis=0)


def covariance(X, mu=None):
    """(mu, C): C = (1/N) (X - mu)^T (X - mu), fp64, both triangles."""
    X64 = np.asarray(X).astype(np.float64)
    if mu is None:
        mu = X64.mean(axis=0)
    Y = X64 - mu
    return mu, (Y.T @ Y) / X64.shape[0]


def canonical_signs(W) -> np.ndarray:
    """Flip each row so that its entry of largest magnitude is positive (lowest
    index among equal magnitudes)."""
    W = np.array(W, dtype=np.float64, copy=True)
    for k in range(W.shape[0]):
        j = int(np.argmax(np.abs(W[k])))  # argmax takes the first of equal values
        if W[k, j] < 0:
            W[k] = -W[k]
    return W


def fit(X, r: int):
    """Principal components of X (N x d): returns (mu[d], W[r x d], lam[d], C[d x d]).

    W holds the r leading eigenvectors of C as rows (decreasing eigenvalue,
    canonical signs); lam holds all d eigenvalues in decreasing order."""
    mu, C = covariance(X)
    vals, vecs = np.linalg.eigh(C)       # ascending eigenvalues, eigenvectors as columns
    order = np.argsort(-vals, kind="stable")
    lam = vals[order]
    W = canonical_signs(vecs[:, order[:r]].T)
    return mu, W, lam, C


def transform(X, mu, W) -> np.ndarray:
    """Projection z_i = W (x_i - mu), fp64 (N x r)."""
    X64 = np.asarray(X).astype(np.float64)
    return (X64 - np.asarray(mu, dtype=np.float64)) @ np.asarray(W, dtype=np.float64).T
