"""GPU parity of the tag statistics of a clustering (Section 4.5) against the oracle.

The GPU takes the partitioned tag lists (hme_partition's outputs); the oracle takes
the raw (labels, tag lists) of every point.  Counts must be identical; the
sparsity ||c(t)||_1 / ||c(t)||_2 is formed from the same integers with correctly
rounded fp64 operations on both sides, so it is held to one ulp.
"""
import dataclasses

import numpy as np
import pytest
import torch

import hme_synth
import oracle

pytestmark = pytest.mark.gpu

hme = pytest.importorskip("paper_1704_06363_gb300.hme")


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    d = torch.device("cuda:0")
    torch.cuda.set_device(d)
    return d


def _zipf_tags(N, V, mean, seed, big_point=None, big_len=0):
    rng = np.random.default_rng(seed)
    lens = rng.poisson(mean, N).astype(np.int64)
    if big_point is not None:
        lens[big_point] = big_len
    tag_off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    w = 1.0 / np.arange(1, V + 1)
    tags = rng.choice(V, int(tag_off[-1]), p=w / w.sum()).astype(np.int32)
    return tag_off, tags


def _gpu_stats(labels, K, tag_off, tags, V, dev, sparsity=True):
    N = labels.shape[0]
    lab = torch.as_tensor(labels, device=dev)
    to = torch.as_tensor(tag_off, device=dev)
    tg = torch.as_tensor(tags if tags.size else np.zeros(1, np.int32), device=dev)
    wp = hme.workspace(hme.HME_OP_PARTITION, N, 1, K, hme.HME_F32, device=dev)
    hist = torch.empty(K, dtype=torch.int64, device=dev)
    offs = torch.empty(K + 1, dtype=torch.int64, device=dev)
    perm = torch.empty(max(N, 1), dtype=torch.int32, device=dev)
    to_out = torch.empty(N + 1, dtype=torch.int64, device=dev)
    tg_out = torch.empty(max(tags.size, 1), dtype=torch.int32, device=dev)
    hme.hme_partition(lab, K, hist, offs, perm, wp, None, to, tg, to_out, tg_out)
    assert hme.hme_sync_status(wp) == hme.HME_OK
    wt = hme.workspace(hme.HME_OP_TAG_HIST, N, V, K, hme.HME_F32, device=dev)
    counts = torch.full((K, V), -7, dtype=torch.int64, device=dev)  # every entry must be written
    sp = torch.full((V,), -1.0, dtype=torch.float64, device=dev) if sparsity else None
    hme.hme_tag_cluster_hist(offs, to_out, tg_out, K, V, counts, wt, sp)
    status = hme.hme_sync_status(wt)
    return status, counts.cpu().numpy(), (sp.cpu().numpy() if sparsity else None)


def _check(labels, K, tag_off, tags, V, dev):
    status, counts, sp = _gpu_stats(labels, K, tag_off, tags, V, dev)
    assert status == hme.HME_OK
    ref_c, ref_s = oracle.tag_cluster_hist(labels, K, tag_off, tags, V)
    assert np.array_equal(counts, ref_c)
    ulp = np.spacing(np.maximum(ref_s, 1.0))
    assert np.all(np.abs(sp - ref_s) <= ulp), float(np.max(np.abs(sp - ref_s) / ulp))
    return counts


@pytest.mark.parametrize("N,K,V", [(3000, 17, 200), (1, 1, 1), (5000, 300, 4096), (777, 64, 50_000)])
def test_tag_hist_parity(dev, N, K, V):
    rng = np.random.default_rng(N + K)
    labels = rng.integers(0, K, N).astype(np.int32)
    tag_off, tags = _zipf_tags(N, V, 3.0, N + V)
    _check(labels, K, tag_off, tags, V, dev)


def test_tag_hist_multi_chunk_and_empty_clusters(dev):
    """One cluster carries > 2 * 65535 tags (several chunks, accumulated with atomics);
    clusters 5..9 are empty (rows of zeros)."""
    N, K, V = 4000, 10, 1000
    rng = np.random.default_rng(4)
    labels = rng.integers(0, 5, N).astype(np.int32)
    labels[17] = 2
    tag_off, tags = _zipf_tags(N, V, 2.0, 9, big_point=17, big_len=150_000)
    counts = _check(labels, K, tag_off, tags, V, dev)
    assert np.all(counts[5:] == 0)


@pytest.mark.parametrize("V", [60_000, 120_000])
def test_tag_hist_large_vocabularies(dev, V):
    """V = 60000: one shared-memory histogram per SM; V = 120000 counters do not fit
    in shared memory: the global-memory counting path."""
    N, K = 6000, 33
    rng = np.random.default_rng(6)
    labels = rng.integers(0, K, N).astype(np.int32)
    tag_off, tags = _zipf_tags(N, V, 4.0, 6)
    _check(labels, K, tag_off, tags, V, dev)


def test_tag_hist_one_tag_fills_a_chunk(dev):
    """70000 copies of one tag on one point: a full chunk of 65535 equal tags (the 16-bit
    field at its maximum) and the rest in a second chunk."""
    N, K, V = 10, 2, 5
    labels = np.array([0, 1] * 5, np.int32)
    lens = np.array([1] * N, np.int64)
    lens[3] = 70_000
    tag_off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    tags = np.full(int(tag_off[-1]), 3, np.int32)
    tags[: tag_off[3]] = 1
    counts = _check(labels, K, tag_off, tags, V, dev)
    assert counts[1, 3] == 70_000 + 3  # point 3, then points 5, 7 and 9 of cluster 1 with one tag 3 each


def test_tag_hist_no_tags(dev):
    N, K, V = 100, 4, 10
    labels = (np.arange(N) % K).astype(np.int32)
    tag_off = np.zeros(N + 1, np.int64)
    _check(labels, K, tag_off, np.zeros(0, np.int32), V, dev)


def test_tag_hist_reports_out_of_range_tag(dev):
    N, K, V = 50, 3, 8
    labels = (np.arange(N) % K).astype(np.int32)
    tag_off = np.arange(N + 1, dtype=np.int64)
    tags = (np.arange(N) % V).astype(np.int32)
    tags[11] = V + 5  # skipped and reported
    status, counts, _ = _gpu_stats(labels, K, tag_off, tags, V, dev)
    assert status == hme.HME_EINVAL
    good = tags.copy()
    keep = np.ones(N, bool)
    keep[11] = False
    ref_c, _ = oracle.tag_cluster_hist(labels, K, tag_off, np.where(keep, good, 0).astype(np.int32), V)
    ref_c[labels[11], 0] -= 1  # the skipped tag was counted as tag 0 in the reference call
    assert np.array_equal(counts, ref_c)


def test_tag_hist_workload4(dev):
    """The tag recipe of the 1.6e7 x 512 workload (Poisson(3) tags, Zipf(1.0) over 20000
    words) at full size, K = 1024 clusters from a seeded labelling."""
    w = hme_synth.WORKLOADS[4]
    tag_off, tags = hme_synth.make_tags(w, device="cpu")
    rng = np.random.default_rng(44)
    labels = rng.integers(0, w.K, w.N).astype(np.int32)
    _check(labels, w.K, tag_off.numpy(), tags.numpy(), w.tag_vocab, dev)


def test_tag_hist_workload4_subsample_of_assignments(dev):
    """Labels from the GPU assign of a workload-4 subsample, tags from the same recipe."""
    w = dataclasses.replace(hme_synth.WORKLOADS[4], N=20_000)
    X, _ = hme_synth.make_features(w, device=dev)
    C = X[torch.arange(0, w.N, w.N // w.K, device=dev)[: w.K]].float().contiguous()
    ws = hme.workspace(hme.HME_OP_ASSIGN, w.N, w.d, w.K, hme.HME_F32, device=dev)
    lab = torch.empty(w.N, dtype=torch.int32, device=dev)
    hme.hme_assign(X, C, lab, ws)
    assert hme.hme_sync_status(ws) == hme.HME_OK
    tag_off, tags = hme_synth.make_tags(w, device="cpu")
    _check(lab.cpu().numpy(), w.K, tag_off.numpy(), tags.numpy(), w.tag_vocab, dev)
