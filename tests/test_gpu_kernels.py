"""GPU parity of each C-ABI entry point against the fp64 oracle (small and ragged shapes)."""
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


def _mixture(N, d, K, dtype, seed, scale=3.0, relu=False, ld=None):
    g = torch.Generator().manual_seed(seed)
    centres = torch.randn(K, d, generator=g) * scale
    comp = torch.randint(0, K, (N,), generator=g)
    X = centres[comp] + torch.randn(N, d, generator=g)
    if relu:
        X.clamp_(min=0)
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    if ld is not None and ld != d:
        buf = torch.zeros(N, ld, dtype=tdt)
        buf[:, :d] = X.to(tdt)
        X = buf[:, :d]
    else:
        X = X.to(tdt)
    return X


def _host(X, dtype):
    return hme_synth.host_array(X.contiguous(), dtype)


def _assign(X, C, dev, mind=True, prepared=False, extra_flags=0):
    N, d = X.shape
    K = C.shape[0]
    Xg = X.to(dev) if X.is_contiguous() else _to_dev_strided(X, dev)
    dt = hme.HME_F32 if X.dtype == torch.float32 else hme.HME_BF16
    ws = hme.workspace(hme.HME_OP_ASSIGN, N, d, K, dt, device=dev)
    lab = torch.full((N,), -1, dtype=torch.int32, device=dev)
    md = torch.empty(N, dtype=torch.float32, device=dev) if mind else None
    obj = torch.zeros(1, dtype=torch.float64, device=dev)
    Cg = C.to(dev)
    if prepared:
        hme.hme_prepare_features(Xg, K, ws)
        hme.hme_assign(Xg, Cg, lab, ws, md, obj, flags=hme.HME_ASSIGN_PREPARED | extra_flags)
    else:
        hme.hme_assign(Xg, Cg, lab, ws, md, obj, flags=extra_flags)
    assert hme.hme_sync_status(ws) == hme.HME_OK
    return lab.cpu().numpy(), (md.cpu().numpy() if mind else None), obj.item()


def _to_dev_strided(X, dev):
    base = X.as_strided((X.shape[0], X.stride(0)), (X.stride(0), 1))
    return base.to(dev)[:, : X.shape[1]]


ASSIGN_CASES = [
    # N, d, K, dtype, ld
    (1000, 128, 16, "f32", None),
    (1000, 128, 16, "bf16", None),
    (777, 33, 5, "f32", None),
    (777, 40, 5, "bf16", None),
    (3000, 130, 300, "f32", None),
    (3000, 130, 300, "bf16", 136),
    (257, 1, 3, "f32", None),
    (129, 64, 1, "f32", None),
    (129, 64, 1, "bf16", None),
    (2000, 512, 1024, "f32", None),
    (2000, 512, 1024, "bf16", None),  # several N-chunks, rows streamed (d > 256): MT = 2, lean scan
    (2000, 256, 4096, "bf16", None),
    (4100, 2048, 64, "f32", None),
    (4100, 2048, 256, "bf16", None),
    (50, 96, 200, "f32", None),
    # the largest K and d the library takes: 64 (fp32) / 128 (bf16, resident rows) N-chunks; 256 k-blocks
    (1500, 64, 16384, "bf16", None),
    (700, 48, 16384, "f32", None),
    (300, 16384, 8, "f32", None),
    (300, 16384, 40, "bf16", 16392),
]


@pytest.mark.parametrize("N,d,K,dtype,ld", ASSIGN_CASES, ids=lambda v: str(v))
def test_assign_parity(dev, N, d, K, dtype, ld):
    X = _mixture(N, d, min(K, 64), dtype, seed=N + d + K, ld=ld)
    C = hme_synth.random_centroids(K, d, seed=K + d, scale=3.0)
    # half of the centres sit on data points so that the nearest one is meaningful
    C[: K // 2] = X[: K // 2].float() if N >= K // 2 else C[: K // 2]
    lab, md, obj = _assign(X, C, dev)
    st = parity.check_assign(_host(X, dtype), dtype, C.numpy(), lab, md, obj)
    assert st["mismatches"] <= st["near_ties"]


# One case per assign kernel variant with at least two row tiles for every
# persistent CTA (one CTA per SM): rows = 2 x SMs x (rows per CTA tile) + 77,
# so each CTA reuses its accumulators and the epilogue's exchange slots across
# tiles, and the last tile is ragged.
#   dtype, d, K, prepared, rows per CTA tile: kernel variant
MULTI_TILE_CASES = [
    ("f32", 256, 64, True, 128),     # three split products, one N-chunk
    ("f32", 256, 64, False, 128),    # fp32 rows split inside the kernel
    ("f32", 200, 600, True, 128),    # three split products, top-three scan over three N-chunks
    ("bf16", 256, 1024, True, 128),  # resident rows, four 256-centre N-chunks (the K = 4096, d = 256 kernel)
    ("bf16", 512, 520, True, 256),   # two row tiles per centre stage, lean scan
    ("bf16", 1024, 256, True, 256),  # two row tiles per centre stage, one 512-column accumulator (K = 256)
]


@pytest.mark.parametrize("dtype,d,K,prepared,bmt", MULTI_TILE_CASES, ids=lambda v: str(v))
def test_assign_parity_several_tiles_per_cta(dev, dtype, d, K, prepared, bmt):
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    N = 2 * sms * bmt + 77
    X = _mixture(N, d, min(K, 64), dtype, seed=N + d + K)
    C = hme_synth.random_centroids(K, d, seed=K + d + 1, scale=3.0)
    C[: K // 2] = X[: K // 2].float()
    lab, md, obj = _assign(X, C, dev, prepared=prepared)
    st = parity.check_assign(_host(X, dtype), dtype, C.numpy(), lab, md, obj)
    assert st["mismatches"] <= st["near_ties"]


# Batches of at most one wave of row tiles spread each tile's centre chunks
# over several CTAs, whose per-row states a second kernel merges.
#   N, d, K, dtype: what the launch does (tiles of 128 rows; 256 for MT = 2)
SLICE_CASES = [
    (256, 256, 4096, "bf16"),   # 2 tiles x 16 slices of one 256-centre chunk
    (256, 256, 4096, "f32"),    # three split products, 16 slices
    (5000, 64, 1100, "bf16"),   # 40 tiles x 3 slices of 2, 2 and 1 chunks (ragged)
    (3000, 512, 1024, "bf16"),  # rows streamed, two row tiles per centre stage: 12 tiles x 4 slices
    (9728, 96, 600, "f32"),     # the most tiles that slice: 76 tiles x 2 slices
    (1, 40, 16384, "bf16"),     # one row against the most centres: 16 slices of 8 chunks
]


@pytest.mark.parametrize("N,d,K,dtype", SLICE_CASES, ids=lambda v: str(v))
def test_small_batch_slices_the_centres(dev, N, d, K, dtype):
    """Near ties between centres of different slices (a copy of each data
    centre 1e-5 away, K/2 columns further on) and exact duplicates (the lowest
    index wins) come out of the slice merge as the oracle has them."""
    X = _mixture(N, d, min(K, 64), dtype, seed=N + K)
    C = hme_synth.random_centroids(K, d, seed=K + 5, scale=3.0)
    m = min(N, K // 4)
    C[:m] = X[:m].float()
    g = torch.Generator().manual_seed(N)
    C[K // 2:K // 2 + m] = C[:m] + 1e-5 * torch.randn(m, d, generator=g)
    C[K - 1] = C[0]  # exact duplicate of centre 0 in the last slice
    lab, md, obj = _assign(X, C, dev)
    st = parity.check_assign(_host(X, dtype), dtype, C.numpy(), lab, md, obj)
    assert st["mismatches"] <= st["near_ties"]
    assert lab[0] == 0  # row 0 sits on centre 0 and on its duplicate K - 1


# HME_ASSIGN_TF32: fp32 features multiplied as tf32 operands (K > 256, rows TMA
# can read); near ties are re-scored on their two candidates, or on all K when
# a third centre is close too.  N, d, K, rows per CTA tile (0: a few tiles)
TF32_CASES = [(2000, 512, 1024, 0), (700, 48, 16384, 0), (3000, 132, 300, 0), (129, 64, 257, 0),
              (0, 200, 600, 256)]


@pytest.mark.parametrize("N,d,K,bmt", TF32_CASES, ids=lambda v: str(v))
@pytest.mark.parametrize("prepared", [False, True])
def test_assign_parity_tf32(dev, N, d, K, bmt, prepared):
    if bmt:  # at least two row tiles per persistent CTA
        N = 2 * torch.cuda.get_device_properties(dev).multi_processor_count * bmt + 77
    X = _mixture(N, d, min(K, 64), "f32", seed=N + d + K + 3)
    C = hme_synth.random_centroids(K, d, seed=K + d + 2, scale=3.0)
    C[: K // 2] = X[: K // 2].float() if N >= K // 2 else C[: K // 2]
    lab, md, obj = _assign(X, C, dev, prepared=prepared, extra_flags=hme.HME_ASSIGN_TF32)
    st = parity.check_assign(_host(X, "f32"), "f32", C.numpy(), lab, md, obj, tf32=True)
    assert st["mismatches"] <= st["near_ties"]


@pytest.mark.parametrize("copies", [2, 3])
def test_assign_tf32_near_ties_are_rescored_exactly(dev, copies):
    """Groups of centres 1e-5 apart: with tf32 operands every such row is a near
    tie, decided by the exact re-score of its two candidates (two copies) or of
    all K (three copies)."""
    N, d, K = 3000, 256, 600
    base = K // copies
    X = _mixture(N, d, 64, "f32", seed=31 + copies)
    C = hme_synth.random_centroids(K, d, seed=4, scale=3.0)
    C[:base] = X[:base].float()
    g = torch.Generator().manual_seed(6)
    for r in range(1, copies):
        C[r * base:(r + 1) * base] = C[:base] + 1e-5 * torch.randn(base, d, generator=g)
    lab, md, obj = _assign(X, C, dev, extra_flags=hme.HME_ASSIGN_TF32)
    st = parity.check_assign(_host(X, "f32"), "f32", C.numpy(), lab, md, obj, tf32=True)
    assert st["mismatches"] <= st["near_ties"]


@pytest.mark.parametrize("dtype,d,K", [("bf16", 256, 32), ("f32", 130, 300)])
def test_assign_prepared_equals_unprepared(dev, dtype, d, K):
    """Where both calls run the same kernel (bf16 features; fp32 with several
    N-chunks), HME_ASSIGN_PREPARED changes nothing: bit-identical results."""
    X = _mixture(2000, d, 32, dtype, seed=5)
    C = hme_synth.random_centroids(K, d, seed=9, scale=3.0)
    a = _assign(X, C, dev, prepared=False)
    b = _assign(X, C, dev, prepared=True)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1]) and a[2] == b[2]


@pytest.mark.parametrize("N,d,K", [(2000, 256, 32), (1001, 36, 7), (513, 2048, 64), (300, 100, 256)])
def test_assign_split_in_kernel_and_prepared_agree(dev, N, d, K):
    """fp32 features, K <= 256: the unprepared call splits rows inside the kernel,
    the prepared one reads the prepared split.  Both meet the oracle's bar; their
    labels agree outside near ties."""
    X = _mixture(N, d, min(K, 32), "f32", seed=N + d)
    C = hme_synth.random_centroids(K, d, seed=9, scale=3.0)
    C[: K // 2] = X[: K // 2].float()
    Xh = _host(X, "f32")
    ref = oracle.assign(Xh, C.numpy(), "f32")
    a = _assign(X, C, dev, prepared=False)
    b = _assign(X, C, dev, prepared=True)
    sa = parity.check_assign(Xh, "f32", C.numpy(), a[0], a[1], a[2], ref=ref)
    sb = parity.check_assign(Xh, "f32", C.numpy(), b[0], b[1], b[2], ref=ref)
    assert sa["mismatches"] <= sa["near_ties"] and sb["mismatches"] <= sb["near_ties"]
    gap = parity.rel_gap(ref[1], ref[2])
    differ = np.nonzero(a[0] != b[0])[0]
    assert np.all(gap[differ] < parity.ASSIGN_GAP)


@pytest.mark.parametrize("N,d,K", [(2000, 256, 32), (1001, 36, 7), (700, 130, 300)])
def test_assign_prepare_out_leaves_the_prepared_split(dev, N, d, K):
    """HME_ASSIGN_PREPARE_OUT: the call's own results are those of a default call
    (bit-identical), and a later HME_ASSIGN_PREPARED call on other centres agrees
    with one after hme_prepare_features (K = 300: the preparation pass; otherwise
    the split written by the assign kernel).  The row norms of the two
    preparations are summed in different orders, so labels may differ only at
    near ties and both meet the oracle's bar."""
    X = _mixture(N, d, min(K, 32), "f32", seed=N + d + 1)
    C1 = hme_synth.random_centroids(K, d, seed=3, scale=3.0)
    C1[: K // 2] = X[: K // 2].float()
    C2 = hme_synth.random_centroids(K, d, seed=4, scale=3.0)
    C2[K // 2:] = X[N - (K - K // 2):].float()
    Xg, C1g, C2g = X.to(dev), C1.to(dev), C2.to(dev)
    ws_out = hme.workspace(hme.HME_OP_ASSIGN, N, d, K, hme.HME_F32, device=dev)
    ws_ref = hme.workspace(hme.HME_OP_ASSIGN, N, d, K, hme.HME_F32, device=dev)

    def run(ws, C, flags):
        lab = torch.full((N,), -1, dtype=torch.int32, device=dev)
        md = torch.empty(N, dtype=torch.float32, device=dev)
        obj = torch.zeros(1, dtype=torch.float64, device=dev)
        hme.hme_assign(Xg, C, lab, ws, md, obj, flags=flags)
        assert hme.hme_sync_status(ws) == hme.HME_OK
        return lab.cpu().numpy(), md.cpu().numpy(), obj.item()

    first = run(ws_out, C1g, hme.HME_ASSIGN_PREPARE_OUT)
    plain = run(ws_ref, C1g, hme.HME_ASSIGN_DEFAULT)
    assert all(np.array_equal(a, b) for a, b in zip(first[:2], plain[:2])) and first[2] == plain[2]
    a = run(ws_out, C2g, hme.HME_ASSIGN_PREPARED)
    hme.hme_prepare_features(Xg, K, ws_ref)
    b = run(ws_ref, C2g, hme.HME_ASSIGN_PREPARED)
    Xh = _host(X, "f32")
    ref = oracle.assign(Xh, C2.numpy(), "f32")
    for r in (a, b):
        st = parity.check_assign(Xh, "f32", C2.numpy(), r[0], r[1], r[2], ref=ref)
        assert st["mismatches"] <= st["near_ties"]
    gap = parity.rel_gap(ref[1], ref[2])
    assert np.all(gap[np.nonzero(a[0] != b[0])[0]] < parity.ASSIGN_GAP)


def test_assign_duplicate_centres_and_zero_rows(dev):
    N, d, K = 600, 64, 8
    X = _mixture(N, d, 4, "f32", seed=3, relu=True)
    X[:50] = 0.0  # all-zero post-ReLU rows
    C = hme_synth.random_centroids(K, d, seed=2)
    C[3] = C[1]  # exact duplicates: ties go to the lower index
    C[5] = C[1]
    lab, md, obj = _assign(X, C, dev)
    assert not np.any((lab == 3) | (lab == 5))
    parity.check_assign(_host(X, "f32"), "f32", C.numpy(), lab, md, obj)


@pytest.mark.parametrize("dtype,K,copies,N", [("f32", 24, 2, 3000), ("bf16", 24, 2, 3000), ("f32", 24, 3, 3000),
                                              ("bf16", 600, 2, 3000), ("f32", 600, 3, 3000), ("f32", 600, 2, 40000),
                                              ("f32", 600, 3, 40000), ("bf16", 600, 2, 40000), ("bf16", 600, 3, 40000),
                                              ("bf16", 1100, 2, 40000)])
def test_assign_near_ties_are_rescored_exactly(dev, dtype, K, copies, N):
    """Groups of centres 1e-5 apart make most rows near ties: the exact re-score decides them.

    Two copies exercise the two-candidate re-score, three the all-K one.  K = 600
    (three N-chunks) on 3000 rows spreads the chunks over CTAs, whose lean scan
    sends every near tie to all K; on 40000 fp32 rows the split kernel's
    top-three scan sends two-candidate near ties to the pair re-score; on 40000
    bf16 rows the lean states name the runner-up's centre when it was another
    state's best (columns in different 16-column groups or epilogue shares), and
    those ties go to the pair re-score too.
    """
    d = 256
    base = K // copies
    X = _mixture(N, d, min(base, 64), dtype, seed=21 + K)
    C = hme_synth.random_centroids(K, d, seed=4, scale=3.0)
    C[:base] = X[:base].float()
    g = torch.Generator().manual_seed(5)
    for r in range(1, copies):
        C[r * base:(r + 1) * base] = C[:base] + 1e-5 * torch.randn(base, d, generator=g)
    lab, md, obj = _assign(X, C, dev)
    st = parity.check_assign(_host(X, dtype), dtype, C.numpy(), lab, md, obj)
    assert st["mismatches"] <= st["near_ties"]


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_small_batch_all_k_rescore_splits_the_centres(dev, dtype):
    """A few near-tie rows against many centres: the all-K re-score splits the
    centres over the blocks (up to 32 slices per row tile here) and merges the
    slices' best per row; labels, distances and the objective match the oracle
    for an assign and for a route of the same batch."""
    B, d, K = 37, 96, 2000
    X = _mixture(B, d, 8, dtype, seed=77)
    C = hme_synth.random_centroids(K, d, seed=78, scale=3.0)
    g = torch.Generator().manual_seed(79)
    C[:B] = X.float()
    for r in (1, 2):  # three centres 1e-5 apart at every row: all-K re-scores
        C[r * B:(r + 1) * B] = C[:B] + 1e-5 * torch.randn(B, d, generator=g)
    lab, md, obj = _assign(X, C, dev)
    st = parity.check_assign(_host(X, dtype), dtype, C.numpy(), lab, md, obj)
    assert st["mismatches"] <= st["near_ties"]
    dt = hme.HME_F32 if dtype == "f32" else hme.HME_BF16
    ws = hme.workspace(hme.HME_OP_ROUTE, B, d, K, dt, device=dev)
    expert = torch.empty(B, dtype=torch.int32, device=dev)
    offs = torch.empty(K + 1, dtype=torch.int64, device=dev)
    order = torch.empty(B, dtype=torch.int32, device=dev)
    hme.hme_route(X.to(dev), C.to(dev), expert, offs, order, ws)
    assert hme.hme_sync_status(ws) == hme.HME_OK
    e = expert.cpu().numpy()
    assert np.array_equal(e, lab)
    parity.check_partition(dict(offsets=offs.cpu().numpy(), perm=order.cpu().numpy()), e, K)



def _full_rescore_rows_per_item(count, K, grid):
    """Rows per work item the all-K re-score picks for a queue of `count` rows:
    the tile with the smaller estimate of max(longest item, all work / grid),
    a 64-row tile costing 16 against 10 for a 32-row one."""
    kt = -(-K // 64)

    def est(fr, cost):
        nt = -(-count // fr)
        ks = min(kt, max(1, grid // max(nt, 1)))
        return max(-(-kt // ks) * cost * grid, nt * kt * cost)

    return 64 if est(64, 16) < est(32, 10) else 32


@pytest.mark.parametrize("dtype,d,ld,K,N,rows_per_item", [("f32", 250, None, 4096, 8000, 64),
                                                          ("bf16", 250, 256, 4096, 8000, 64),
                                                          ("bf16", 256, None, 4096, 8000, 64),
                                                          ("f32", 250, None, 600, 300, 32),
                                                          ("bf16", 256, None, 4096, 200, 32)])
def test_all_k_rescore_long_and_short_queues(dev, dtype, d, ld, K, N, rows_per_item):
    """Three centres 1e-5 apart around every data row send nearly every row to
    the all-K re-score.  A long queue runs in 64-row work items, a short one in
    32-row items; d = 250 (centre rows not 16 bytes apart) stages the centres
    one element at a time, d = 256 in 16-byte loads.  Labels, distances and the
    objective match the oracle."""
    copies = 3
    base = K // copies
    nb = min(base, N)  # data rows that become centres (with two copies each)
    X = _mixture(N, d, min(base, 64), dtype, seed=91 + K + d, ld=ld)
    C = hme_synth.random_centroids(K, d, seed=92, scale=3.0)
    C[:nb] = X[:nb].float()
    g = torch.Generator().manual_seed(93)
    for r in range(1, copies):
        C[r * base:r * base + nb] = C[:nb] + 1e-5 * torch.randn(nb, d, generator=g)
    Xg = X.to(dev) if X.is_contiguous() else _to_dev_strided(X, dev)
    dt = hme.HME_F32 if dtype == "f32" else hme.HME_BF16
    ws = hme.workspace(hme.HME_OP_ASSIGN, N, d, K, dt, device=dev)
    lab = torch.full((N,), -1, dtype=torch.int32, device=dev)
    md = torch.empty(N, dtype=torch.float32, device=dev)
    obj = torch.zeros(1, dtype=torch.float64, device=dev)
    hme.hme_assign(Xg, C.to(dev), lab, ws, md, obj)
    assert hme.hme_sync_status(ws) == hme.HME_OK
    # workspace header, 32-bit words: [1] rows queued for a pair re-score, [3] for all K
    all_k = int(ws[:16].view(torch.int32).cpu()[3])
    assert all_k >= N // 2
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    assert _full_rescore_rows_per_item(all_k, K, 4 * sms) == rows_per_item  # the tile this case is for
    st = parity.check_assign(_host(X, dtype), dtype, C.numpy(), lab.cpu().numpy(), md.cpu().numpy(), obj.item())
    assert st["mismatches"] <= st["near_ties"]

def test_route_reuses_prepared_features(dev):
    N, d, K = 4000, 128, 16
    X = _mixture(N, d, K, "f32", seed=8)
    C = hme_synth.random_centroids(K, d, seed=8, scale=3.0)
    C[:8] = X[:8]
    Xg, Cg = X.to(dev), C.to(dev)
    ws = hme.workspace(hme.HME_OP_ASSIGN, N, d, K, hme.HME_F32, device=dev)
    outs = []
    for flags in (hme.HME_ASSIGN_DEFAULT, hme.HME_ASSIGN_PREPARED):
        if flags == hme.HME_ASSIGN_PREPARED:
            hme.hme_prepare_features(Xg, K, ws)
        e = torch.empty(N, dtype=torch.int32, device=dev)
        o = torch.empty(K + 1, dtype=torch.int64, device=dev)
        r = torch.empty(N, dtype=torch.int32, device=dev)
        hme.hme_route(Xg, Cg, e, o, r, ws, flags=flags)
        assert hme.hme_sync_status(ws) == hme.HME_OK
        outs.append((e.cpu(), o.cpu(), r.cpu()))
    assert all(torch.equal(a, b) for a, b in zip(*outs))


def test_assign_empty_input(dev):
    X = torch.empty(0, 64, dtype=torch.float32)
    C = hme_synth.random_centroids(4, 64, seed=1)
    ws = hme.workspace(hme.HME_OP_ASSIGN, 0, 64, 4, hme.HME_F32, device=dev)
    lab = torch.empty(0, dtype=torch.int32, device=dev)
    obj = torch.full((1,), 7.0, dtype=torch.float64, device=dev)
    hme.hme_assign(X.to(dev), C.to(dev), lab, ws, None, obj)
    assert hme.hme_sync_status(ws) == hme.HME_OK and obj.item() == 0.0


UPDATE_CASES = [
    (1000, 128, 16, "f32", False),
    (1000, 128, 16, "bf16", False),
    (3001, 130, 37, "f32", True),
    (3001, 136, 37, "bf16", True),
    (5000, 2048, 64, "f32", False),
    (5000, 256, 700, "bf16", True),
    (300, 20, 500, "f32", True),  # more clusters than points: reseeds run out of rows
    (20000, 64, 90, "f32", True),  # about 18 empty clusters: one-pass selection
    (20000, 64, 400, "bf16", True),  # about 80 empty clusters: the general path
]


@pytest.mark.parametrize("N,d,K,dtype,holes", UPDATE_CASES, ids=lambda v: str(v))
def test_update_parity(dev, N, d, K, dtype, holes):
    X = _mixture(N, d, min(K, 50), dtype, seed=N * 7 + K)
    g = torch.Generator().manual_seed(K)
    w = torch.arange(1, K + 1, dtype=torch.float64) ** -1.1
    labels = torch.multinomial(w, N, replacement=True, generator=g).to(torch.int32)
    if holes:  # force empty clusters
        labels[(labels % 5) == 2] = 0
    mind = (torch.rand(N, generator=g) * 10).float()
    mind[:7] = 5.0  # ties in the farthest-point order
    C0 = hme_synth.random_centroids(K, d, seed=3)
    dt = hme.HME_F32 if dtype == "f32" else hme.HME_BF16
    ws = hme.workspace(hme.HME_OP_ASSIGN, N, d, K, dt, device=dev)
    Cg = C0.to(dev)
    counts = torch.empty(K, dtype=torch.int64, device=dev)
    nres = torch.full((1,), -1, dtype=torch.int32, device=dev)
    J = torch.zeros(1, dtype=torch.float64, device=dev)
    hme.hme_update_centroids(X.to(dev), labels.to(dev), mind.to(dev), Cg, ws, counts, nres, J)
    assert hme.hme_sync_status(ws) == hme.HME_OK
    parity.check_objective(J.item(), _host(X, dtype), dtype, C0.numpy(), labels.numpy())
    Cref, cref, nref = oracle.update(_host(X, dtype), labels.numpy(), mind.double().numpy(), C0.numpy(), dtype)
    assert np.array_equal(counts.cpu().numpy(), cref)
    assert nres.item() == nref
    parity.check_centres(Cg.cpu().numpy(), Cref)
    # re-seeded centres are exact copies of rows
    empty = np.nonzero(cref == 0)[0]
    assert np.array_equal(Cg.cpu().numpy()[empty], Cref[empty])


@pytest.mark.parametrize("N,d,K,dtype,frac", [(4000, 256, 24, "f32", 0.05), (4000, 136, 24, "bf16", 0.3),
                                              (3001, 130, 300, "f32", 0.02), (2000, 64, 40, "bf16", 1.0)])
def test_update_incremental_matches_oracle(dev, N, d, K, dtype, frac):
    """An update from the previous call's state, reading only rows whose label changed,
    gives the oracle's centres, counts and objective for the new labels."""
    X = _mixture(N, d, min(K, 30), dtype, seed=N + K + 7)
    g = torch.Generator().manual_seed(11)
    lab0 = torch.randint(0, K, (N,), generator=g, dtype=torch.int32)
    lab0[lab0 == 5] = 6  # cluster 5 empty at first: re-seeded, then filled
    lab1 = lab0.clone()
    moved = torch.rand(N, generator=g) < frac
    lab1[moved] = torch.randint(0, K, (int(moved.sum()),), generator=g, dtype=torch.int32)
    lab1[lab1 == 7] = 8  # cluster 7 empties in the second call
    mind = (torch.rand(N, generator=g) * 10).float()
    C0 = hme_synth.random_centroids(K, d, seed=6)
    dt = hme.HME_F32 if dtype == "f32" else hme.HME_BF16
    ws = hme.workspace(hme.HME_OP_ASSIGN, N, d, K, dt, device=dev)
    Xg, md = X.to(dev), mind.to(dev)
    Cg = C0.to(dev)
    counts = torch.empty(K, dtype=torch.int64, device=dev)
    nres = torch.zeros(1, dtype=torch.int32, device=dev)
    J = torch.zeros(1, dtype=torch.float64, device=dev)
    hme.hme_update_centroids(Xg, lab0.to(dev), md, Cg, ws, counts, nres, J)
    assert hme.hme_sync_status(ws) == hme.HME_OK
    C1 = Cg.cpu().numpy()
    Xh = _host(X, dtype)
    hme.hme_update_centroids(Xg, lab1.to(dev), md, Cg, ws, counts, nres, J, prev_labels=lab0.to(dev))
    assert hme.hme_sync_status(ws) == hme.HME_OK
    Cref, cref, nref = oracle.update(Xh, lab1.numpy(), mind.double().numpy(), C1, dtype)
    assert np.array_equal(counts.cpu().numpy(), cref) and nres.item() == nref
    parity.check_centres(Cg.cpu().numpy(), Cref)
    parity.check_objective(J.item(), Xh, dtype, C1, lab1.numpy())


PART_CASES = [(0, 4), (1, 1), (31, 7), (1000, 64), (100003, 1000), (70000, 4096), (50000, 1), (12345, 16384)]


@pytest.mark.parametrize("N,K", PART_CASES, ids=lambda v: str(v))
def test_partition_bit_exact(dev, N, K):
    g = torch.Generator().manual_seed(N + K)
    w = torch.arange(1, K + 1, dtype=torch.float64) ** -1.0
    labels = torch.multinomial(w, max(N, 1), replacement=True, generator=g).to(torch.int32)[:N]
    ws = hme.workspace(hme.HME_OP_PARTITION, N, 1, K, hme.HME_F32, device=dev)
    hist = torch.empty(K, dtype=torch.int64, device=dev)
    offs = torch.empty(K + 1, dtype=torch.int64, device=dev)
    perm = torch.empty(N, dtype=torch.int32, device=dev)
    sl = torch.empty(N, dtype=torch.int32, device=dev)
    hme.hme_partition(labels.to(dev), K, hist, offs, perm, ws, sl)
    assert hme.hme_sync_status(ws) == hme.HME_OK
    parity.check_partition(dict(hist=hist.cpu().numpy(), offsets=offs.cpu().numpy(), perm=perm.cpu().numpy(),
                                sorted_labels=sl.cpu().numpy()), labels.numpy(), K)


# Labels spread evenly over K buckets (the shape of converged K-means labels,
# unlike the Zipf draws above), several sort chunks per tile, one and two
# tiles per SM (K from 2048 on: one), every digit-pass split up to K = 16384.
UNIFORM_PART_CASES = [(2_000_000, 300), (1_000_001, 600), (1_500_000, 2048), (3_000_000, 4096), (1_500_000, 5000),
                      (777_777, 8192), (1_300_000, 16384)]


@pytest.mark.parametrize("N,K", UNIFORM_PART_CASES, ids=lambda v: str(v))
def test_partition_uniform_labels(dev, N, K):
    g = torch.Generator().manual_seed(N ^ K)
    labels = torch.randint(0, K, (N,), generator=g, dtype=torch.int32)
    ws = hme.workspace(hme.HME_OP_PARTITION, N, 1, K, hme.HME_F32, device=dev)
    hist = torch.empty(K, dtype=torch.int64, device=dev)
    offs = torch.empty(K + 1, dtype=torch.int64, device=dev)
    perm = torch.empty(N, dtype=torch.int32, device=dev)
    sl = torch.empty(N, dtype=torch.int32, device=dev)
    hme.hme_partition(labels.to(dev), K, hist, offs, perm, ws, sl)
    assert hme.hme_sync_status(ws) == hme.HME_OK
    parity.check_partition(dict(hist=hist.cpu().numpy(), offsets=offs.cpu().numpy(), perm=perm.cpu().numpy(),
                                sorted_labels=sl.cpu().numpy()), labels.numpy(), K)


def test_partition_many_buckets_drops_bad_labels(dev):
    """Labels outside [0, K) are counted nowhere, reported, and left out of
    the order; the valid ones keep their stable order."""
    N, K = 600_000, 1000
    g = torch.Generator().manual_seed(7)
    labels = torch.randint(-3, K + 3, (N,), generator=g, dtype=torch.int32)
    ws = hme.workspace(hme.HME_OP_PARTITION, N, 1, K, hme.HME_F32, device=dev)
    hist = torch.empty(K, dtype=torch.int64, device=dev)
    offs = torch.empty(K + 1, dtype=torch.int64, device=dev)
    perm = torch.full((N,), -1, dtype=torch.int32, device=dev)
    hme.hme_partition(labels.to(dev), K, hist, offs, perm, ws)
    assert hme.hme_sync_status(ws) == hme.HME_EINVAL
    lab = labels.numpy()
    ok = (lab >= 0) & (lab < K)
    assert np.array_equal(hist.cpu().numpy(), np.bincount(lab[ok], minlength=K))
    nv = int(ok.sum())
    ref = np.nonzero(ok)[0][np.argsort(lab[ok], kind="stable")]
    assert np.array_equal(perm.cpu().numpy()[:nv], ref)


def test_partition_tags_and_misaligned_labels(dev):
    N, K = 20001, 33
    w = hme_synth.WORKLOADS[4].with_rows(N)
    tag_off, tags = hme_synth.make_tags(w)
    g = torch.Generator().manual_seed(1)
    full = torch.randint(0, K, (N + 1,), generator=g, dtype=torch.int32)
    labels_d = full.to(dev)[1:]  # 4-byte offset: exercises the unaligned staging path
    ws = hme.workspace(hme.HME_OP_PARTITION, N, 1, K, hme.HME_F32, device=dev)
    hist = torch.empty(K, dtype=torch.int64, device=dev)
    offs = torch.empty(K + 1, dtype=torch.int64, device=dev)
    perm = torch.empty(N, dtype=torch.int32, device=dev)
    too = torch.empty(N + 1, dtype=torch.int64, device=dev)
    tgo = torch.empty(tags.numel(), dtype=torch.int32, device=dev)
    hme.hme_partition(labels_d, K, hist, offs, perm, ws, None, tag_off.to(dev), tags.to(dev), too, tgo)
    assert hme.hme_sync_status(ws) == hme.HME_OK
    parity.check_partition(dict(hist=hist.cpu().numpy(), offsets=offs.cpu().numpy(), perm=perm.cpu().numpy(),
                                tag_off=too.cpu().numpy(), tags=tgo.cpu().numpy()),
                           full[1:].numpy(), K, tag_off.numpy(), tags.numpy())


def test_partition_bad_label_reports_einval(dev):
    labels = torch.tensor([0, 1, 9, 2, -3, 1], dtype=torch.int32, device=dev)
    K = 3
    ws = hme.workspace(hme.HME_OP_PARTITION, 6, 1, K, hme.HME_F32, device=dev)
    hist = torch.empty(K, dtype=torch.int64, device=dev)
    offs = torch.empty(K + 1, dtype=torch.int64, device=dev)
    perm = torch.full((6,), -1, dtype=torch.int32, device=dev)
    hme.hme_partition(labels, K, hist, offs, perm, ws)
    assert hme.hme_sync_status(ws) == hme.HME_EINVAL
    assert hist.cpu().tolist() == [1, 2, 1]  # the valid labels are still counted
    assert perm.cpu().tolist()[:4] == [0, 1, 5, 3]


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_route_parity(dev, dtype):
    B, d, K = 5000, 192, 40
    Q = _mixture(B, d, K, dtype, seed=11)
    C = hme_synth.random_centroids(K, d, seed=12, scale=3.0)
    C[:20] = Q[:20].float()
    dt = hme.HME_F32 if dtype == "f32" else hme.HME_BF16
    ws = hme.workspace(hme.HME_OP_ROUTE, B, d, K, dt, device=dev)
    expert = torch.empty(B, dtype=torch.int32, device=dev)
    offs = torch.empty(K + 1, dtype=torch.int64, device=dev)
    order = torch.empty(B, dtype=torch.int32, device=dev)
    hme.hme_route(Q.to(dev), C.to(dev), expert, offs, order, ws)
    assert hme.hme_sync_status(ws) == hme.HME_OK
    e = expert.cpu().numpy()
    parity.check_assign(_host(Q, dtype), dtype, C.numpy(), e)
    parity.check_partition(dict(offsets=offs.cpu().numpy(), perm=order.cpu().numpy()), e, K)


def test_route_replayed_graph_reads_fresh_data(dev):
    """Repeated small routes with the same arguments replay a captured graph:
    the third and fourth calls, on new batch contents and new centres at the
    same addresses, route them exactly as a first call does."""
    B, d, K = 256, 256, 4096
    ws = hme.workspace(hme.HME_OP_ROUTE, B, d, K, hme.HME_BF16, device=dev)
    Q = torch.empty(B, d, dtype=torch.bfloat16, device=dev)
    C = torch.empty(K, d, dtype=torch.float32, device=dev)
    expert = torch.empty(B, dtype=torch.int32, device=dev)
    offs = torch.empty(K + 1, dtype=torch.int64, device=dev)
    order = torch.empty(B, dtype=torch.int32, device=dev)
    for call in range(4):
        Qh = _mixture(B, d, 16, "bf16", seed=100 + call)
        Ch = hme_synth.random_centroids(K, d, seed=200 + call, scale=3.0)
        Ch[:B // 2] = Qh[:B // 2].float()
        Q.copy_(Qh)
        C.copy_(Ch)
        before = hme.hme_launch_count()
        hme.hme_route(Q, C, expert, offs, order, ws)
        assert hme.hme_sync_status(ws) == hme.HME_OK
        assert hme.hme_launch_count() > before  # replays count their kernels too
        e = expert.cpu().numpy()
        parity.check_assign(_host(Qh, "bf16"), "bf16", Ch.numpy(), e)
        parity.check_partition(dict(offsets=offs.cpu().numpy(), perm=order.cpu().numpy()), e, K)


@pytest.mark.parametrize("N,d,K,dtype,method", [
    (10000, 128, 16, "f32", hme.HME_INIT_KMEANSPP),
    (3000, 64, 9, "bf16", hme.HME_INIT_KMEANSPP),
    (20000, 96, 8, "f32", hme.HME_INIT_KMEANSPP_SUBSAMPLE),
    (7, 5, 7, "f32", hme.HME_INIT_KMEANSPP),
])
def test_kmeanspp_matches_oracle(dev, N, d, K, dtype, method):
    X = _mixture(N, d, K, dtype, seed=N + K)
    dt = hme.HME_F32 if dtype == "f32" else hme.HME_BF16
    ws = hme.workspace(hme.HME_OP_INIT, N, d, K, dt, device=dev)
    C = torch.empty(K, d, dtype=torch.float32, device=dev)
    for seed in (0, 1, 2**63 + 5):
        hme.hme_kmeans_init(X.to(dev), K, seed, method, C, ws)
        assert hme.hme_sync_status(ws) == hme.HME_OK
        Cref, _ = oracle.kmeanspp(_host(X, dtype), K, seed, method == hme.HME_INIT_KMEANSPP_SUBSAMPLE, dtype)
        assert np.array_equal(C.cpu().numpy(), Cref)


def test_bounded_wait_reports_timeout_and_context_survives(dev):
    ws = torch.empty(256, dtype=torch.uint8, device=dev)
    hme.hme_debug_bounded_wait(2_000_000, ws)  # 2 ms on a barrier nothing completes
    assert hme.hme_sync_status(ws) == hme.HME_ETIMEOUT
    x = torch.arange(10, device=dev).sum().item()  # the context is still usable
    assert x == 45


def test_launch_counter_moves(dev):
    before = hme.hme_launch_count()
    X = _mixture(300, 32, 4, "f32", seed=1)
    _assign(X, hme_synth.random_centroids(4, 32, seed=1), dev)
    assert hme.hme_launch_count() - before >= 3


@pytest.mark.parametrize("dtype,d,K", [("f32", 256, 32), ("bf16", 256, 300), ("f32", 128, 600), ("f32", 130, 40)])
def test_assign_rows_in_chunks_equals_one_call(dev, dtype, d, K):
    """hme_assign_rows over consecutive row ranges (ragged, one of a single
    row) gives the labels and distances of one hme_assign call, bit for bit
    (the per-row arithmetic is the same), and the preparation the chunks leave
    (HME_ASSIGN_PREPARE_OUT) serves a later prepared call like one left by a
    single call."""
    N = 5000
    X = _mixture(N, d, min(K, 32), dtype, seed=d + K)
    C = hme_synth.random_centroids(K, d, seed=K, scale=3.0)
    C[: K // 2] = X[: K // 2].float()
    C2 = hme_synth.random_centroids(K, d, seed=K + 1, scale=3.0)
    C2[K // 2:] = X[N - (K - K // 2):].float()
    Xg, Cg, C2g = X.to(dev), C.to(dev), C2.to(dev)
    dt = hme.HME_F32 if dtype == "f32" else hme.HME_BF16
    out = []
    for chunked in (True, False):
        ws = hme.workspace(hme.HME_OP_ASSIGN, N, d, K, dt, device=dev)
        lab = torch.full((N,), -1, dtype=torch.int32, device=dev)
        md = torch.empty(N, dtype=torch.float32, device=dev)
        if chunked:
            bounds = [0, 1234, 1235, 4000, N]
            for r0, r1 in zip(bounds, bounds[1:]):
                hme.hme_assign_rows(Xg, r0, r1, Cg, lab, ws, md, flags=hme.HME_ASSIGN_PREPARE_OUT)
        else:
            hme.hme_assign(Xg, Cg, lab, ws, md, flags=hme.HME_ASSIGN_PREPARE_OUT)
        lab2 = torch.full((N,), -1, dtype=torch.int32, device=dev)
        md2 = torch.empty(N, dtype=torch.float32, device=dev)
        hme.hme_assign(Xg, C2g, lab2, ws, md2, flags=hme.HME_ASSIGN_PREPARED)
        assert hme.hme_sync_status(ws) == hme.HME_OK
        out.append([t.cpu().numpy() for t in (lab, md, lab2, md2)])
    for a, b in zip(*out):
        assert np.array_equal(a, b)
    st = parity.check_assign(_host(X, dtype), dtype, C.numpy(), out[0][0], out[0][1])
    assert st["mismatches"] <= st["near_ties"]


def test_assign_rows_rejects_ranges_outside_the_set(dev):
    X = _mixture(100, 32, 4, "f32", seed=1).to(dev)
    C = hme_synth.random_centroids(4, 32, seed=1).to(dev)
    ws = hme.workspace(hme.HME_OP_ASSIGN, 100, 32, 4, hme.HME_F32, device=dev)
    lab = torch.empty(100, dtype=torch.int32, device=dev)
    for r0, r1 in ((-1, 5), (10, 5), (90, 101)):
        with pytest.raises(hme.HmeError) as ei:
            hme.hme_assign_rows(X, r0, r1, C, lab, ws)
        assert ei.value.code == hme.HME_EINVAL
