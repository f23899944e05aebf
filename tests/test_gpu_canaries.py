"""Guard bands around every output of the C ABI (host-side bounds check).

Each output array (and the workspace) is a view into a larger buffer whose
leading and trailing bands hold a fixed byte pattern; after ragged-size calls
of hme_assign, hme_update_centroids, hme_partition (with tag lists) and
hme_route the bands must be unchanged.  This catches any kernel that writes
past the end (or before the start) of an array it was given.
"""
import numpy as np
import pytest
import torch

import hme_synth

pytestmark = pytest.mark.gpu

hme = pytest.importorskip("paper_1704_06363_gb300.hme")

GUARD = 4096  # bytes of pattern on each side
PATTERN = 0xA5


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    d = torch.device("cuda:0")
    torch.cuda.set_device(d)
    return d


class Guarded:
    """numel elements of dtype inside GUARD bytes of pattern on each side."""

    def __init__(self, numel, dtype, dev, shape=None):
        es = torch.empty(0, dtype=dtype).element_size()
        self.g = GUARD // es
        self.raw = torch.full((numel * es + 2 * GUARD,), PATTERN, dtype=torch.uint8, device=dev)
        self.t = self.raw.view(dtype)[self.g:self.g + numel]
        if shape is not None:
            self.t = self.t.view(*shape)

    def intact(self):
        r = self.raw.cpu().numpy()
        return bool(np.all(r[:GUARD] == PATTERN) and np.all(r[-GUARD:] == PATTERN))


def _ws(op, N, d, K, dt, dev):
    return Guarded(hme.hme_workspace_bytes(op, N, d, K, dt), torch.uint8, dev)


@pytest.mark.parametrize("N", [1, 129, 4100])
@pytest.mark.parametrize("dtype,d,K", [("f32", 130, 37), ("bf16", 256, 300), ("f32", 64, 600)])
def test_outputs_keep_their_guard_bands(dev, N, dtype, d, K):
    g = torch.Generator().manual_seed(N + d + K)
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    dt = hme.HME_F32 if dtype == "f32" else hme.HME_BF16
    X = (torch.randn(N, d, generator=g) * 3).to(tdt).to(dev)
    C = Guarded(K * d, torch.float32, dev, (K, d))
    C.t.copy_(hme_synth.random_centroids(K, d, seed=K, scale=3.0).to(dev))
    C.t[: min(K, N)] = X[: min(K, N)].float()

    # assign (prepared, as in a Lloyd loop)
    ws = _ws(hme.HME_OP_ASSIGN, N, d, K, dt, dev)
    labels = Guarded(N, torch.int32, dev)
    mind = Guarded(N, torch.float32, dev)
    obj = Guarded(1, torch.float64, dev)
    hme.hme_assign(X, C.t, labels.t, ws.t, mind.t, obj.t, flags=hme.HME_ASSIGN_PREPARE_OUT)
    hme.hme_assign(X, C.t, labels.t, ws.t, mind.t, obj.t, flags=hme.HME_ASSIGN_PREPARED)
    assert hme.hme_sync_status(ws.t) == hme.HME_OK
    # centre update: full pass, then incremental from other labels
    counts = Guarded(K, torch.int64, dev)
    nres = Guarded(1, torch.int32, dev)
    J = Guarded(1, torch.float64, dev)
    hme.hme_update_centroids(X, labels.t, mind.t, C.t, ws.t, counts.t, nres.t, J.t)
    prev = labels.t.clone()
    labels.t.copy_(torch.randint(0, K, (N,), generator=g, dtype=torch.int32).to(dev))
    hme.hme_update_centroids(X, labels.t, mind.t, C.t, ws.t, counts.t, nres.t, J.t, prev_labels=prev)
    assert hme.hme_sync_status(ws.t) == hme.HME_OK
    # partition with tag lists
    w4 = hme_synth.WORKLOADS[4].with_rows(N)
    tag_off, tags = hme_synth.make_tags(w4, device=dev)
    T = tags.numel()
    wp = _ws(hme.HME_OP_PARTITION, N, 1, K, dt, dev)
    hist = Guarded(K, torch.int64, dev)
    offs = Guarded(K + 1, torch.int64, dev)
    perm = Guarded(N, torch.int32, dev)
    srt = Guarded(N, torch.int32, dev)
    too = Guarded(N + 1, torch.int64, dev)
    tgo = Guarded(max(T, 1), torch.int32, dev)
    hme.hme_partition(labels.t, K, hist.t, offs.t, perm.t, wp.t, srt.t, tag_off, tags, too.t, tgo.t)
    assert hme.hme_sync_status(wp.t) == hme.HME_OK
    # route
    wr = _ws(hme.HME_OP_ROUTE, N, d, K, dt, dev)
    expert = Guarded(N, torch.int32, dev)
    roffs = Guarded(K + 1, torch.int64, dev)
    order = Guarded(N, torch.int32, dev)
    hme.hme_route(X, C.t, expert.t, roffs.t, order.t, wr.t)
    assert hme.hme_sync_status(wr.t) == hme.HME_OK
    torch.cuda.synchronize()
    named = dict(C=C, ws_assign=ws, labels=labels, mind=mind, objective=obj, counts=counts, n_reseeded=nres,
                 J=J, ws_partition=wp, hist=hist, offsets=offs, perm=perm, sorted_labels=srt, tag_off_out=too,
                 tags_out=tgo, ws_route=wr, expert=expert, route_offsets=roffs, order=order)
    broken = [k for k, v in named.items() if not v.intact()]
    assert not broken, f"guard bands overwritten: {broken}"
