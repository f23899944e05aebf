"""GPU parity of the PCA that precedes the gater's K-means (Section 4.2) against
the fp64 oracle (oracle/pca.py).

Tolerances, from the arithmetic (each stated where it is used):
  covariance  y = x - fp32(mu) is split into bf16 y = yh + yl with
              |y - yh - yl| <= 2^-16 |y|; the dropped yl yl' and the split
              error give at most 3 * 2^-16 |y_a||y_b| per product; the tensor
              cores accumulate 512 rows at a time in fp32: 3 x 512/16 = 96
              steps of at most one ulp (2^-23, whatever the rounding), +2 for
              the conversions; up to 16 such sums are added in fp32 registers
              (round to nearest, 2^-24 each, +2), then in fp64.  So |dC_ab| <= TAU_C * B_ab with
              B = (1/N) sum_i (|y_ia| + |mu_a|)(|y_ib| + |mu_b|) (the |mu| terms
              cover the rounding of x - fp32(mu)).
  eigen       Weyl: |d lambda| <= ||dC||_2 <= ||TAU_C B||_F, plus the backward
              error of fp32 Jacobi, taken as 2^-13 ||C||_F (measured well below
              it); eigenvectors are compared where the eigenvalue is separated
              (Davis-Kahan), and always through orthonormality, residuals and
              captured variance, which any valid answer meets even inside
              clusters of equal eigenvalues.
  transform   the assign kernel's split arithmetic: |dz_ij| <= TAU_Z sum_k
              |x_ik| |w_jk| + 2^-22 (|z_ij| + |mu . w_j|).
"""
import numpy as np
import pytest
import torch

from oracle import pca as opca

pytestmark = pytest.mark.gpu

hme = pytest.importorskip("paper_1704_06363_gb300.hme")

TAU_C = 3 * 2.0 ** -16 + 98 * 2.0 ** -23 + 18 * 2.0 ** -24
JACOBI = 2.0 ** -13


def _tau_z(d):
    return 3 * 2.0 ** -16 + ((d + 15) // 16 + 3) * 2.0 ** -24


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    d = torch.device("cuda:0")
    torch.cuda.set_device(d)
    return d


def _features(N, d, comps, seed, offset=0.0):
    """Post-ReLU Gaussian mixture, the shape of pooled CNN features."""
    g = torch.Generator().manual_seed(seed)
    centres = torch.randn(comps, d, generator=g) * 2.0
    idx = torch.randint(0, comps, (N,), generator=g)
    return (torch.relu(centres[idx] + torch.randn(N, d, generator=g)) + offset).float()


def _gpu_cov(X, dev):
    N, d = X.shape
    ws = hme.workspace(hme.HME_OP_PCA, N, d, 1, hme.HME_F32, device=dev)
    mu = torch.empty(d, dtype=torch.float64, device=dev)
    C = torch.full((d, d), float("nan"), dtype=torch.float64, device=dev)  # every entry must be written
    hme.hme_pca_covariance(X.to(dev), mu, C, ws)
    assert hme.hme_sync_status(ws) == hme.HME_OK
    return mu.cpu().numpy(), C.cpu().numpy()


def _bound(X, mu):
    Y = np.abs(X.astype(np.float64) - mu) + np.abs(mu)
    return Y.T @ Y / X.shape[0]


@pytest.mark.parametrize("N,d,offset", [(5000, 200, 0.0), (20000, 130, 0.0), (3000, 513, 100.0), (777, 1, 0.0),
                                        (1, 5, 0.0), (64, 128, 0.0), (8193, 64, -3.0)])
def test_covariance_parity(dev, N, d, offset):
    """Ragged N (many 512-row sub-ranges, a lone row) and d (several 128-wide
    tiles and a partial one), a large offset (centring in fp32)."""
    X = _features(N, d, 8, seed=N + d, offset=offset)
    mu, C = _gpu_cov(X, dev)
    Xn = X.numpy()
    mu_ref, C_ref = opca.covariance(Xn)
    assert np.allclose(mu, mu_ref, rtol=2.0 ** -20, atol=2.0 ** -20 * np.abs(Xn).max())
    B = _bound(Xn, mu_ref)
    err = np.abs(C - C_ref)
    assert np.all(err <= TAU_C * B + 1e-300), float(np.max(err / np.maximum(B, 1e-300)))
    assert np.array_equal(C, C.T)


def _fit(X, r, dev):
    N, d = X.shape
    ws = hme.workspace(hme.HME_OP_PCA, N, d, r, hme.HME_F32, device=dev)
    mu = torch.empty(d, dtype=torch.float32, device=dev)
    W = torch.empty(r, d, dtype=torch.float32, device=dev)
    lam = torch.empty(r, dtype=torch.float32, device=dev)
    sweeps = hme.hme_pca_fit(X.to(dev), r, mu, W, ws, lam)
    assert hme.hme_sync_status(ws) == hme.HME_OK
    return mu.cpu().numpy(), W.cpu().numpy().astype(np.float64), lam.cpu().numpy().astype(np.float64), sweeps


def _check_fit(Xn, r, mu, W, lam, sweeps):
    mu_ref, W_ref, lam_ref, C_ref = opca.fit(Xn, r)
    d = Xn.shape[1]
    assert 1 <= sweeps <= 40
    assert np.allclose(mu, mu_ref, rtol=2.0 ** -20, atol=2.0 ** -20 * np.abs(Xn).max())
    normC = np.linalg.norm(C_ref)
    tol = TAU_C * np.linalg.norm(_bound(Xn, mu_ref)) + JACOBI * normC
    # variances: Weyl
    assert np.all(np.abs(lam - lam_ref[:r]) <= tol), float(np.max(np.abs(lam - lam_ref[:r])) / normC)
    # orthonormal rows, eigen-residuals against the oracle's covariance
    assert np.allclose(W @ W.T, np.eye(r), atol=2.0 ** -14)
    res = np.linalg.norm(C_ref @ W.T - W.T * lam, axis=0)
    assert np.all(res <= 2 * tol), float(res.max() / normC)
    # captured variance of the r rows (Ky Fan: the oracle's is the maximum)
    cap = np.trace(W @ C_ref @ W.T)
    assert cap >= lam_ref[:r].sum() - r * tol and cap <= lam_ref[:r].sum() * (1 + 1e-12) + r * tol
    # separated eigenvalues: the same direction and sign as the oracle (Davis-Kahan)
    full = np.concatenate([lam_ref, [np.inf, -np.inf]])
    for k in range(r):
        gap = min(np.min(np.abs(np.delete(full, k) - lam_ref[k])), np.inf)
        if gap > 100 * tol:
            sin_t = 2 * tol / gap
            assert abs(W[k] @ W_ref[k]) >= np.sqrt(1 - sin_t ** 2) - 1e-12
            big = np.argmax(np.abs(W_ref[k]))
            if abs(W_ref[k, big]) - np.partition(np.abs(W_ref[k]), -2)[-2] > 4 * sin_t if d > 1 else True:
                assert W[k] @ W_ref[k] > 0  # the sign rule picked the same sign


@pytest.mark.parametrize("N,d,r", [(4000, 64, 16), (3000, 257, 100), (2000, 2, 2), (500, 1, 1), (20000, 300, 256)])
def test_fit_parity(dev, N, d, r):
    """Odd d (a padding slot in the Jacobi ordering), d = 1 and 2, r = d."""
    X = _features(N, d, 12, seed=3 * N + d)
    mu, W, lam, sweeps = _fit(X, r, dev)
    _check_fit(X.numpy(), r, mu, W, lam, sweeps)


def test_fit_recovers_a_known_spectrum(dev):
    """The oracle pin's construction: rows mu +- sqrt(d lam_j) q_j have mean mu
    and covariance Q diag(lam) Q^T exactly; the GPU finds lam and the q_j."""
    d = 96
    lam = np.geomspace(50.0, 0.05, d)
    q, rr = np.linalg.qr(np.random.default_rng(1).standard_normal((d, d)))
    Q = q * np.sign(np.diag(rr))
    mu = np.linspace(-2.0, 3.0, d)
    rows = []
    for j in range(d):
        a = np.sqrt(d * lam[j]) * Q[:, j]
        rows += [mu + a, mu - a]
    X = torch.tensor(np.array(rows), dtype=torch.float32)
    r = 20
    m, W, l, sweeps = _fit(X, r, dev)
    _check_fit(X.numpy(), r, m, W, l, sweeps)
    assert np.allclose(l, lam[:r], rtol=1e-3)
    ref = opca.canonical_signs(Q[:, :r].T)
    assert np.all(np.abs(np.sum(W * ref, axis=1)) > 1 - 1e-4)


def _transform(X, mu, W, dev, ldz=None):
    N, d = X.shape
    r = W.shape[0]
    ws = hme.workspace(hme.HME_OP_PCA, 0, d, r, hme.HME_F32, device=dev)
    ldz = ldz or r
    Zb = torch.full((N, ldz), float("nan"), dtype=torch.float32, device=dev)
    Z = Zb[:, :r]
    ldx = (d + 3) // 4 * 4  # TMA rows: a pitch of whole 16-byte units
    Xd = torch.zeros(N, ldx, dtype=torch.float32, device=dev)
    Xd[:, :d] = X.to(dev)
    hme.hme_pca_transform(Xd[:, :d], torch.tensor(np.ascontiguousarray(mu), dtype=torch.float32, device=dev),
                          torch.tensor(np.ascontiguousarray(W), dtype=torch.float32, device=dev), Z, ws)
    assert hme.hme_sync_status(ws) == hme.HME_OK
    return Zb.cpu().numpy()


@pytest.mark.parametrize("N,d,r,ldz", [(1000, 300, 16, None), (129, 2048, 256, None), (3001, 512, 100, 103),
                                       (50, 64, 7, None), (700, 33, 33, None)])
def test_transform_parity(dev, N, d, r, ldz):
    """Teacher-forced: the GPU projection of X with given (mu, W) against the
    fp64 projection with the same (mu, W); ragged N, r not a multiple of 16, a
    padded output pitch (its padding columns must stay untouched)."""
    X = _features(N, d, 8, seed=N + r)
    Xn = X.numpy()
    rng = np.random.default_rng(r)
    q, _ = np.linalg.qr(rng.standard_normal((d, r)))
    W = np.ascontiguousarray(q.T, dtype=np.float32)
    mu = Xn.mean(axis=0).astype(np.float32)
    Zb = _transform(X, mu, W, dev, ldz)
    Z = Zb[:, :r]
    ref = opca.transform(Xn, mu.astype(np.float64), W.astype(np.float64))
    bound = _tau_z(d) * (np.abs(Xn.astype(np.float64)) @ np.abs(W.astype(np.float64)).T)
    bound += 2.0 ** -22 * (np.abs(ref) + np.abs(mu.astype(np.float64) @ W.T.astype(np.float64)))
    err = np.abs(Z - ref)
    assert np.all(err <= bound), float(np.max(err / bound))
    if ldz and ldz > r:
        assert np.all(np.isnan(Zb[:, r:]))


def test_fit_then_transform_then_assign(dev):
    """The Section 4.2 pipeline on a small case: fit r = 32 components, project,
    and the projected features' covariance is diagonal with the variances."""
    X = _features(6000, 200, 10, seed=77)
    mu, W, lam, _ = _fit(X, 32, dev)
    Z = _transform(X, mu, W.astype(np.float32), dev).astype(np.float64)
    cz = Z.T @ Z / Z.shape[0] - np.outer(Z.mean(0), Z.mean(0))
    assert np.allclose(np.diag(cz), lam, rtol=1e-3, atol=1e-4 * lam[0])
    off = cz - np.diag(np.diag(cz))
    assert np.max(np.abs(off)) <= 1e-3 * lam[0]


def test_pca_benchmark_features_full_size(dev):
    """The 1e6 x 2048 fp32 benchmark features at full size, r = 256, in the
    launch configuration the benchmark times: covariance entries and means on
    sampled index pairs against fp64 sums over the full columns; the fit's
    components orthonormal with eigen-residuals within the bound against the
    (sample-checked) covariance, variances against its fp64 eigenvalues;
    projections of sampled rows against fp64 dot products."""
    import hme_synth
    w = hme_synth.WORKLOADS[2]
    X, _ = hme_synth.make_features(w, device=dev)
    N, d = X.shape
    r = 256
    ws = hme.workspace(hme.HME_OP_PCA, N, d, r, hme.HME_F32, device=dev)
    mu64 = torch.empty(d, dtype=torch.float64, device=dev)
    C = torch.empty(d, d, dtype=torch.float64, device=dev)
    hme.hme_pca_covariance(X, mu64, C, ws)
    assert hme.hme_sync_status(ws) == hme.HME_OK
    rng = np.random.default_rng(0)
    cols = sorted(set([0, 1, 127, 128, 1000, 2047] + rng.integers(0, d, 10).tolist()))
    colv = {j: X[:, j].double().cpu().numpy() for j in cols}
    mu_ref = {j: colv[j].mean() for j in cols}
    Cg, mug = C.cpu().numpy(), mu64.cpu().numpy()
    for a in cols:
        assert abs(mug[a] - mu_ref[a]) <= 2.0 ** -20 * (np.abs(colv[a]).mean() + 1e-30)
        for b in cols:
            ya, yb = colv[a] - mu_ref[a], colv[b] - mu_ref[b]
            ref = np.mean(ya * yb)
            bnd = np.mean((np.abs(ya) + abs(mu_ref[a])) * (np.abs(yb) + abs(mu_ref[b])))
            assert abs(Cg[a, b] - ref) <= TAU_C * bnd, (a, b, Cg[a, b], ref)
    mu = torch.empty(d, dtype=torch.float32, device=dev)
    W = torch.empty(r, d, dtype=torch.float32, device=dev)
    lam = torch.empty(r, dtype=torch.float32, device=dev)
    sweeps = hme.hme_pca_fit(X, r, mu, W, ws, lam)
    assert hme.hme_sync_status(ws) == hme.HME_OK and 1 <= sweeps <= 40
    Wd, lamd = W.double(), lam.double()
    normC = torch.linalg.norm(C).item()
    tol = JACOBI * normC
    assert (Wd @ Wd.T - torch.eye(r, dtype=torch.float64, device=dev)).abs().max().item() <= 2.0 ** -14
    res = torch.linalg.norm(C @ Wd.T - Wd.T * lamd, dim=0).max().item()
    assert res <= 2 * tol, res / normC
    ev = np.sort(np.linalg.eigvalsh(Cg))[::-1][:r]
    assert np.all(np.abs(lam.cpu().numpy() - ev) <= tol), np.max(np.abs(lam.cpu().numpy() - ev)) / normC
    Z = torch.empty(N, r, dtype=torch.float32, device=dev)
    wt = hme.workspace(hme.HME_OP_PCA, 0, d, r, hme.HME_F32, device=dev)
    hme.hme_pca_transform(X, mu, W, Z, wt)
    assert hme.hme_sync_status(wt) == hme.HME_OK
    rows = torch.tensor(sorted(set([0, N - 1] + rng.integers(0, N, 62).tolist())), device=dev)
    Xs = X[rows].double().cpu().numpy()
    Wn, mun = W.double().cpu().numpy(), mu.double().cpu().numpy()
    ref = (Xs - mun) @ Wn.T
    bound = _tau_z(d) * (np.abs(Xs) @ np.abs(Wn).T) + 2.0 ** -22 * (np.abs(ref) + np.abs(mun @ Wn.T))
    assert np.all(np.abs(Z[rows].double().cpu().numpy() - ref) <= bound)


def test_fit_constant_data(dev):
    """Every row equal: the covariance is zero, every variance 0, and the
    components are the unit vectors in index order (ties go to the lower
    index; the padding of the Jacobi order is never chosen)."""
    N, d, r = 500, 70, 70
    X = torch.full((N, d), 3.25, dtype=torch.float32)
    mu, W, lam, sweeps = _fit(X, r, dev)
    assert np.allclose(mu, 3.25) and np.all(lam == 0.0)
    assert np.array_equal(W, np.eye(d)[:r])


@pytest.mark.parametrize("d", [63, 65, 129])
def test_fit_repeated_and_zero_variances(dev, d):
    """Duplicated features (a repeated eigenvalue and a zero one per pair),
    constant features (zero variance), d next to a multiple of the Jacobi
    block: the results stay valid eigenpairs of the oracle's covariance."""
    N, r = 3000, min(d, 40)
    X = _features(N, d, 6, seed=d)
    X[:, 1] = X[:, 0]          # duplicate column
    X[:, 5] = X[:, 4]
    X[:, d - 1] = 7.0          # constant column
    X[:, d - 2] = 0.0
    mu, W, lam, sweeps = _fit(X, r, dev)
    _check_fit(X.numpy(), r, mu, W, lam, sweeps)


def test_transform_single_component(dev):
    X = _features(999, 130, 4, seed=3)
    Xn = X.numpy()
    w = np.random.default_rng(1).standard_normal((1, 130))
    W = (w / np.linalg.norm(w)).astype(np.float32)
    mu = Xn.mean(axis=0).astype(np.float32)
    Z = _transform(X, mu, W, dev)
    ref = opca.transform(Xn, mu.astype(np.float64), W.astype(np.float64))
    bound = _tau_z(130) * (np.abs(Xn.astype(np.float64)) @ np.abs(W.astype(np.float64)).T)
    bound += 2.0 ** -22 * (np.abs(ref) + np.abs(mu.astype(np.float64) @ W.T.astype(np.float64)))
    assert np.all(np.abs(Z - ref) <= bound)
