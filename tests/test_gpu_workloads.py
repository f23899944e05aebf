"""GPU parity on the five workloads (seeded synthetic stand-ins for the paper's feature sets).

- Workload 1 in full: the GPU k-means++ seeding equals the oracle's, then ten Lloyd
  iterations teacher-forced (both sides get the GPU's C_t each iteration), then the
  partition.
- Workloads 2-5 on row subsamples of the same recipes (several tiles and a ragged
  tail): seeding, two teacher-forced iterations, the partition (workload 4 moves its
  tag lists) and the route of a fresh batch.
- Workloads 2-5 at full size, in the launch configuration bench.py times: sampled
  rows against the oracle, exact counts and partition (workload 4 moves its tag
  lists), sampled cluster means.  Workloads 3 and 4 are the two whose feature
  matrices hold more than 2^31 elements.
"""
import dataclasses

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


def _dt(w):
    return hme.HME_F32 if w.dtype == "f32" else hme.HME_BF16


class Lloyd:
    """GPU state for one feature set (the calls bench.py makes)."""

    def __init__(self, w, X, dev):
        self.w, self.X, self.dev = w, X, dev
        N, d, K = X.shape[0], w.d, w.K
        self.ws = hme.workspace(hme.HME_OP_ASSIGN, N, d, K, _dt(w), device=dev)
        self.labels = torch.empty(N, dtype=torch.int32, device=dev)
        self.mind = torch.empty(N, dtype=torch.float32, device=dev)
        self.obj = torch.zeros(1, dtype=torch.float64, device=dev)
        self.J = torch.zeros(1, dtype=torch.float64, device=dev)
        self.counts = torch.empty(K, dtype=torch.int64, device=dev)
        self.nres = torch.zeros(1, dtype=torch.int32, device=dev)
        self.prev = None  # labels of the previous centre update: later updates are incremental
        hme.hme_prepare_features(X, K, self.ws)

    def init(self, seed, method):
        wi = hme.workspace(hme.HME_OP_INIT, self.X.shape[0], self.w.d, self.w.K, _dt(self.w), device=self.dev)
        C = torch.empty(self.w.K, self.w.d, dtype=torch.float32, device=self.dev)
        hme.hme_kmeans_init(self.X, self.w.K, seed, method, C, wi)
        assert hme.hme_sync_status(wi) == hme.HME_OK
        return C

    def assign(self, C):
        hme.hme_assign(self.X, C, self.labels, self.ws, self.mind, self.obj, flags=hme.HME_ASSIGN_PREPARED)
        assert hme.hme_sync_status(self.ws) == hme.HME_OK

    def update(self, C):
        hme.hme_update_centroids(self.X, self.labels, self.mind, C, self.ws, self.counts, self.nres, self.J,
                                 prev_labels=self.prev)
        assert hme.hme_sync_status(self.ws) == hme.HME_OK
        self.prev = self.labels.clone()


def _teacher_forced(w, Xh, L, C, iters):
    """Each iteration both sides start from the GPU's C_t."""
    stats = []
    for _ in range(iters):
        C_t = C.cpu().numpy()
        L.assign(C)
        lab = L.labels.cpu().numpy()
        md = L.mind.cpu().numpy()
        st = parity.check_assign(Xh, w.dtype, C_t, lab, md, L.obj.item())
        L.update(C)
        parity.check_objective(L.J.item(), Xh, w.dtype, C_t, lab)
        Cref, cref, nref = oracle.update(Xh, lab, md.astype(np.float64), C_t, w.dtype)
        assert np.array_equal(L.counts.cpu().numpy(), cref)
        assert L.nres.item() == nref
        parity.check_centres(C.cpu().numpy(), Cref)
        stats.append(st)
    return stats


def _partition(labels, K, dev, tag_off=None, tags=None):
    N = labels.numel()
    ws = hme.workspace(hme.HME_OP_PARTITION, N, 1, K, hme.HME_F32, device=dev)
    out = dict(hist=torch.empty(K, dtype=torch.int64, device=dev),
               offsets=torch.empty(K + 1, dtype=torch.int64, device=dev),
               perm=torch.empty(N, dtype=torch.int32, device=dev),
               sorted_labels=torch.empty(N, dtype=torch.int32, device=dev))
    extra = {}
    if tag_off is not None:
        extra = dict(tag_off=torch.empty(N + 1, dtype=torch.int64, device=dev),
                     tags=torch.empty(max(tags.numel(), 1), dtype=torch.int32, device=dev))
        hme.hme_partition(labels, K, out["hist"], out["offsets"], out["perm"], ws, out["sorted_labels"],
                          tag_off, tags, extra["tag_off"], extra["tags"])
    else:
        hme.hme_partition(labels, K, out["hist"], out["offsets"], out["perm"], ws, out["sorted_labels"])
    assert hme.hme_sync_status(ws) == hme.HME_OK
    res = {k: v.cpu().numpy() for k, v in out.items()}
    if extra:
        res["tag_off"] = extra["tag_off"].cpu().numpy()
        res["tags"] = extra["tags"].cpu().numpy()[: tags.numel()]
    return res


def test_workload1_full(dev):
    w = hme_synth.WORKLOADS[1]
    X, comp = hme_synth.make_features(w, device="cpu")
    Xh = hme_synth.host_array(X, w.dtype)
    Xg = X.to(dev)
    L = Lloyd(w, Xg, dev)
    C = L.init(w.seed, hme.HME_INIT_KMEANSPP)
    C0_ref, _ = oracle.kmeanspp(Xh, w.K, w.seed, False, w.dtype)
    assert np.array_equal(C.cpu().numpy(), C0_ref)
    stats = _teacher_forced(w, Xh, L, C, w.iters)
    assert all(s["mismatches"] <= s["near_ties"] for s in stats)
    L.assign(C)
    lab = L.labels.cpu().numpy()
    parity.check_partition(_partition(L.labels, w.K, dev), lab, w.K)
    # free running, reported not gated: the oracle's own 10 iterations from the same seed
    _, lab_free, _, _, _ = oracle.lloyd(Xh, C0_ref, w.iters, w.dtype)
    agree = float(np.mean(lab_free == lab))
    print(f"workload 1 free-running label agreement with the oracle: {agree:.6f}")


SUBSAMPLES = {2: 20_000, 3: 12_000, 4: 20_000, 5: 12_000}


@pytest.mark.parametrize("wid", [2, 3, 4, 5])
def test_workload_subsample(dev, wid):
    w = hme_synth.WORKLOADS[wid].with_rows(SUBSAMPLES[wid])
    X, _ = hme_synth.make_features(w, device="cpu")
    Xh = hme_synth.host_array(X, w.dtype)
    Xg = X.to(dev)
    L = Lloyd(w, Xg, dev)
    method = hme.HME_INIT_KMEANSPP_SUBSAMPLE if w.init_subsample else hme.HME_INIT_KMEANSPP
    seed = 1000 + wid
    C = L.init(seed, method)
    C0_ref, _ = oracle.kmeanspp(Xh, w.K, seed, w.init_subsample, w.dtype)
    assert np.array_equal(C.cpu().numpy(), C0_ref)
    stats = _teacher_forced(w, Xh, L, C, 2)
    assert all(s["mismatches"] <= s["near_ties"] for s in stats)
    L.assign(C)
    lab = L.labels.cpu().numpy()
    if w.tags:
        tag_off, tags = hme_synth.make_tags(w)
        got = _partition(L.labels, w.K, dev, tag_off.to(dev), tags.to(dev))
        parity.check_partition(got, lab, w.K, tag_off.numpy(), tags.numpy())
    else:
        parity.check_partition(_partition(L.labels, w.K, dev), lab, w.K)
    # route a fresh batch from the same recipe (other seed) with the final centres
    B = 3001
    Q, _ = hme_synth.make_features(dataclasses.replace(w, seed=w.seed + 50, N=B), device="cpu")
    wr = hme.workspace(hme.HME_OP_ROUTE, B, w.d, w.K, _dt(w), device=dev)
    expert = torch.empty(B, dtype=torch.int32, device=dev)
    offs = torch.empty(w.K + 1, dtype=torch.int64, device=dev)
    order = torch.empty(B, dtype=torch.int32, device=dev)
    hme.hme_route(Q.to(dev), C, expert, offs, order, wr)
    assert hme.hme_sync_status(wr) == hme.HME_OK
    e = expert.cpu().numpy()
    parity.check_assign(hme_synth.host_array(Q, w.dtype), w.dtype, C.cpu().numpy(), e)
    parity.check_partition(dict(offsets=offs.cpu().numpy(), perm=order.cpu().numpy()), e, w.K)


def _gather_rows(Xg, rows, dtype):
    idx = torch.as_tensor(rows, dtype=torch.int64, device=Xg.device)
    return hme_synth.host_array(Xg.index_select(0, idx), dtype)


@pytest.mark.parametrize("wid", [2, 3, 4, 5])
def test_workload_full_size_sampled(dev, wid):
    w = hme_synth.WORKLOADS[wid]
    X, _ = hme_synth.make_features(w, device=dev)
    L = Lloyd(w, X, dev)
    C = L.init(1234 + w.seed, hme.HME_INIT_KMEANSPP_SUBSAMPLE)
    rng = np.random.default_rng(wid)
    for it in range(2):
        C_t = C.cpu().numpy()
        L.assign(C)
        lab = L.labels.cpu().numpy()
        rows = np.sort(rng.choice(w.N, 2048, replace=False))
        # the last rows of the matrix too: past 2^31 elements for workloads 3 and 4
        rows = np.unique(np.concatenate([rows, np.arange(w.N - 5, w.N)]))
        Xs = _gather_rows(X, rows, w.dtype)
        st = parity.check_assign(Xs, w.dtype, C_t, lab[rows], L.mind.cpu().numpy()[rows])
        assert st["mismatches"] <= st["near_ties"]
        L.update(C)
        counts = L.counts.cpu().numpy()
        assert np.array_equal(counts, np.bincount(lab, minlength=w.K))
        # sampled cluster means: the oracle on the gathered members of a few
        # clusters (of at most 300,000 members, to bound the host copy)
        Cg = C.cpu().numpy()
        eligible = np.nonzero((counts > 0) & (counts <= 300_000))[0]
        pick = rng.choice(eligible, min(4, eligible.size), replace=False)
        for k in pick:
            members = np.nonzero(lab == k)[0]
            Xk = _gather_rows(X, members, w.dtype)
            Cref, _, _ = oracle.update(Xk, np.zeros(members.size, np.int32), None, C_t[k:k + 1], w.dtype)
            parity.check_centres(Cg[k:k + 1], Cref)
    # the partition of the full label vector, bit-exact (workload 4 with its tag lists)
    if w.tags:
        tag_off, tags = hme_synth.make_tags(w, device=dev)
        got = _partition(L.labels, w.K, dev, tag_off, tags)
        parity.check_partition(got, lab, w.K, tag_off.cpu().numpy(), tags.cpu().numpy())
    else:
        got = _partition(L.labels, w.K, dev)
        parity.check_partition(got, lab, w.K)
