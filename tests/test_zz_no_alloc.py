"""hme_partition_noalloc: the expert partition for callers that cannot allocate
device memory (no workspace; its scratch is a fixed array inside the library).

Its outputs must equal hme_partition's bit for bit, on consecutive calls that
reuse the shared array with different sizes (so nothing from an earlier call
may leak into a later one), including a size that forces longer tiles so that
the per-tile counts fit in the array.  Collected last on purpose.
"""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

hme = pytest.importorskip("paper_1704_06363_gb300.hme")


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_1704_06363_gb300 import _build
    _build.build()
    d = torch.device("cuda:0")
    torch.cuda.set_device(d)
    return d


def _labels(N, K, seed, dev):
    g = torch.Generator().manual_seed(seed)
    w = torch.arange(1, K + 1, dtype=torch.float64) ** -1.0
    return torch.multinomial(w, N, replacement=True, generator=g).to(torch.int32).to(dev)


def _with_workspace(labels, K, dev):
    N = labels.numel()
    ws = hme.workspace(hme.HME_OP_PARTITION, N, 1, K, hme.HME_F32, device=dev)
    hist = torch.empty(K, dtype=torch.int64, device=dev)
    offs = torch.empty(K + 1, dtype=torch.int64, device=dev)
    perm = torch.empty(N, dtype=torch.int32, device=dev)
    sl = torch.empty(N, dtype=torch.int32, device=dev)
    hme.hme_partition(labels, K, hist, offs, perm, ws, sl)
    assert hme.hme_sync_status(ws) == hme.HME_OK
    return [t.cpu() for t in (hist, offs, perm, sl)]


def _without_workspace(labels, K, dev):
    N = labels.numel()
    hist = torch.full((K,), -1, dtype=torch.int64, device=dev)
    offs = torch.full((K + 1,), -1, dtype=torch.int64, device=dev)
    perm = torch.full((N,), -1, dtype=torch.int32, device=dev)
    sl = torch.full((N,), -1, dtype=torch.int32, device=dev)
    status = torch.full((1,), -7, dtype=torch.int32, device=dev)
    hme.hme_partition_noalloc(labels, K, hist, offs, perm, sl, status)
    torch.cuda.synchronize(dev)
    assert status.item() == 0
    return [t.cpu() for t in (hist, offs, perm, sl)]


def test_noalloc_matches_hme_partition_on_consecutive_calls(dev):
    cases = [
        (100_003, 1000, 1),
        (5_003, 7, 2),             # smaller, right after a larger call
        (20_000_000, 16384, 3),    # counts only fit with longer tiles
        (1, 1, 4),
    ]
    for N, K, seed in cases:
        labels = _labels(N, K, seed, dev)
        ref = _with_workspace(labels, K, dev)
        got = _without_workspace(labels, K, dev)
        for name, a, b in zip(("hist", "offsets", "perm", "sorted_labels"), ref, got):
            assert torch.equal(a, b), f"N={N} K={K}: {name} differs from hme_partition"
        assert np.array_equal(ref[2].numpy(), np.argsort(labels.cpu().numpy(), kind="stable"))


def test_noalloc_rejects_sizes_beyond_its_limits(dev):
    labels = _labels(10, 3, 5, dev)
    hist = torch.empty(3, dtype=torch.int64, device=dev)
    offs = torch.empty(4, dtype=torch.int64, device=dev)
    perm = torch.empty(10, dtype=torch.int32, device=dev)
    for K in (0, 16385):
        with pytest.raises(hme.HmeError) as ei:
            hme.hme_partition_noalloc(labels, K, hist, offs, perm)
        assert ei.value.code == hme.HME_EINVAL


def test_noalloc_reports_a_bad_label(dev):
    labels = torch.tensor([0, 1, 5, 2, 1], dtype=torch.int32, device=dev)
    hist = torch.empty(3, dtype=torch.int64, device=dev)
    offs = torch.empty(4, dtype=torch.int64, device=dev)
    perm = torch.empty(5, dtype=torch.int32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    hme.hme_partition_noalloc(labels, 3, hist, offs, perm, None, status)
    torch.cuda.synchronize(dev)
    assert status.item() == 1 and hist.cpu().tolist() == [1, 2, 1]
