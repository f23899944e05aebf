"""GPU parity of Lloyd's iterations on a feature set streamed from page-locked host
memory (hme_kmeans_stream) against the oracle, one iteration per call so that both
sides start each iteration from the GPU's centres (teacher forcing), with ragged
chunks, both feature types and empty clusters re-seeded from host rows."""
import numpy as np
import pytest
import torch

import hme_synth
import oracle
from tests import parity

pytestmark = pytest.mark.gpu

hme = pytest.importorskip("paper_1704_06363_gb300.hme")


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    d = torch.device("cuda:0")
    torch.cuda.set_device(d)
    return d


def _mixture(N, d, comps, dtype, seed):
    g = torch.Generator().manual_seed(seed)
    centres = torch.randn(comps, d, generator=g) * 3.0
    idx = torch.randint(0, comps, (N,), generator=g)
    X = torch.relu(centres[idx] + torch.randn(N, d, generator=g))
    return X.to(torch.bfloat16) if dtype == "bf16" else X


class Streamed:
    def __init__(self, X_host, K, chunk, dev):
        self.X = X_host
        N, d = X_host.shape
        dt = hme.HME_F32 if X_host.dtype == torch.float32 else hme.HME_BF16
        self.ws = hme.workspace(hme.HME_OP_STREAM, chunk, d, K, dt, device=dev)
        self.labels = torch.empty(N, dtype=torch.int32, device=dev)
        self.mind = torch.empty(N, dtype=torch.float32, device=dev)
        self.obj = torch.zeros(4, dtype=torch.float64, device=dev)
        self.counts = torch.empty(K, dtype=torch.int64, device=dev)
        self.nres = torch.zeros(1, dtype=torch.int32, device=dev)
        self.K, self.chunk = K, chunk

    def run(self, C, iters):
        hme.hme_kmeans_stream(self.X, self.K, iters, self.chunk, C, self.labels, self.mind, self.ws, self.obj,
                              self.counts, self.nres)
        assert hme.hme_sync_status(self.ws) == hme.HME_OK


@pytest.mark.parametrize("N,d,K,dtype,chunk", [(20001, 64, 12, "f32", 3000), (9000, 72, 40, "bf16", 2500),
                                               (5000, 300, 300, "f32", 4096)])
def test_stream_teacher_forced(dev, N, d, K, dtype, chunk):
    X = _mixture(N, d, min(K, 16), dtype, seed=N + K)
    Xp = X.pin_memory()
    Xh = hme_synth.host_array(X, dtype)
    C = X[torch.randperm(N, generator=torch.Generator().manual_seed(3))[:K]].float().contiguous().to(dev)
    S = Streamed(Xp, K, chunk, dev)
    for _ in range(2):
        C_t = C.cpu().numpy()
        S.run(C, 1)
        lab = S.labels.cpu().numpy()
        st = parity.check_assign(Xh, dtype, C_t, lab, S.mind.cpu().numpy())
        assert st["mismatches"] <= st["near_ties"]
        parity.check_objective(S.obj[0].item(), Xh, dtype, C_t, lab)
        Cref, cref, nref = oracle.update(Xh, lab, S.mind.cpu().numpy().astype(np.float64), C_t, dtype)
        assert np.array_equal(S.counts.cpu().numpy(), cref)
        assert S.nres.item() == nref
        parity.check_centres(C.cpu().numpy(), Cref)


def test_stream_reseeds_empty_clusters_from_host_rows(dev):
    """60 centres on 6 well separated groups: most clusters go empty and take the
    farthest rows, read in place from page-locked host memory."""
    N, d, K = 6000, 32, 60
    X = _mixture(N, d, 6, "f32", seed=5)
    Xh = hme_synth.host_array(X, "f32")
    C = (X[:K].float() + 0.01).contiguous().to(dev)
    C[10:] = 1000.0  # far from every row: empty after the first assign
    S = Streamed(X.pin_memory(), K, 1777, dev)
    C_t = C.cpu().numpy()
    S.run(C, 1)
    lab = S.labels.cpu().numpy()
    Cref, cref, nref = oracle.update(Xh, lab, S.mind.cpu().numpy().astype(np.float64), C_t, "f32")
    assert nref > 0 and S.nres.item() == nref
    assert np.array_equal(S.counts.cpu().numpy(), cref)
    parity.check_centres(C.cpu().numpy(), Cref)


def test_stream_matches_in_hbm_lloyd(dev):
    """Three iterations streamed vs three in-HBM iterations (hme_assign + full
    hme_update_centroids) from the same centres: the same labels but for rows whose
    two best centres tie to within the tolerance, centres within the centre
    tolerance (only the fp64 summation order differs)."""
    N, d, K = 12000, 128, 24
    X = _mixture(N, d, 24, "f32", seed=9)
    C0 = X[:K].float().contiguous().to(dev)
    S = Streamed(X.pin_memory(), K, 5000, dev)
    Cs = C0.clone()
    S.run(Cs, 3)
    Xg = X.to(dev)
    ws = hme.workspace(hme.HME_OP_ASSIGN, N, d, K, hme.HME_F32, device=dev)
    lab = torch.empty(N, dtype=torch.int32, device=dev)
    mind = torch.empty(N, dtype=torch.float32, device=dev)
    Ch = C0.clone()
    for _ in range(3):
        C_last = Ch.cpu().numpy()  # the centres the final labels were assigned against
        hme.hme_assign(Xg, Ch, lab, ws, mind)
        hme.hme_update_centroids(Xg, lab, mind, Ch, ws)
    assert hme.hme_sync_status(ws) == hme.HME_OK
    a, b = S.labels.cpu().numpy(), lab.cpu().numpy()
    differ = np.nonzero(a != b)[0]
    if differ.size:
        _, d1, d2, _ = oracle.assign(hme_synth.host_array(X, "f32")[differ], C_last, "f32")
        assert np.all(parity.rel_gap(d1, d2) < parity.ASSIGN_GAP)
    parity.check_centres(Cs.cpu().numpy(), Ch.cpu().numpy().astype(np.float64))


def test_stream_accepts_device_memory_and_rejects_pageable_host(dev):
    N, d, K = 3000, 16, 5
    X = _mixture(N, d, 5, "f32", seed=2)
    C = X[:K].float().contiguous().to(dev)
    S = Streamed(X.to(dev), K, 1000, dev)
    S.run(C, 1)
    Sh = Streamed(X.clone(), K, 1000, dev)  # ordinary (pageable) host memory
    with pytest.raises(hme.HmeError):
        Sh.run(C, 1)
