"""CPU-side checks of the C ABI: the library builds, loads without a GPU, exports
every entry point that include/hme.h declares, and rejects bad arguments on the
host before any CUDA call is made."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "hme.h")


@pytest.fixture(scope="module")
def lib():
    from paper_1704_06363_gb300 import _build
    path = _build.build()
    return ctypes.CDLL(path)


def declared_entry_points():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"HME_API\s+[\w\s\*]+?\b(hme_\w+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_entry_points()
    for required in ["hme_kmeans_init", "hme_assign", "hme_update_centroids", "hme_partition", "hme_route",
                     "hme_workspace_bytes", "hme_last_error", "hme_sync_status", "hme_prepare_features"]:
        assert required in names


def test_library_exports_every_declared_symbol(lib):
    for name in declared_entry_points():
        assert hasattr(lib, name), f"{name} declared in hme.h but not exported"


def test_workspace_sizes(lib):
    f = lib.hme_workspace_bytes
    f.restype = ctypes.c_size_t
    f.argtypes = [ctypes.c_int32, ctypes.c_int64, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32]
    # fp32 features carry their bf16 split (4 bytes per element) in the workspace
    assert f(1, 1_000_000, 2048, 64, 0) >= 1_000_000 * 2048 * 4
    assert f(1, 1_000_000, 2048, 64, 1) < 1_000_000 * 2048  # bf16: no copy of X
    assert f(2, 50_000_000, 256, 4096, 1) > 0
    assert f(2, 0, 1, 1, 0) > 0
    assert f(1, 10, 0, 4, 0) == 0  # d = 0 rejected
    assert f(1, 10, 4, 0, 0) == 0  # K = 0 rejected
    assert f(1, 10, 4, 4, 7) == 0  # unknown dtype
    assert f(1, 2**31, 4, 4, 0) == 0


def test_host_validation_rejects_before_launch(lib):
    lib.hme_assign.restype = ctypes.c_int
    lib.hme_last_error.restype = ctypes.c_char_p
    p = ctypes.c_void_p
    args = [p(16), ctypes.c_int64(10), ctypes.c_int32(8), ctypes.c_int64(8), ctypes.c_int32(0), p(16),
            ctypes.c_int32(4), ctypes.c_int32(0), p(16), None, None, p(256), ctypes.c_size_t(1 << 30), None]
    bad_k = list(args)
    bad_k[6] = ctypes.c_int32(0)
    assert lib.hme_assign(*bad_k) == 1 and b"K" in lib.hme_last_error()
    bad_ld = list(args)
    bad_ld[3] = ctypes.c_int64(4)
    assert lib.hme_assign(*bad_ld) == 1
    bad_ws = list(args)
    bad_ws[11] = p(257)
    assert lib.hme_assign(*bad_ws) == 1 and b"aligned" in lib.hme_last_error()
    small_ws = list(args)
    small_ws[12] = ctypes.c_size_t(16)
    assert lib.hme_assign(*small_ws) == 2  # HME_ENOMEM
    bf16_misaligned = list(args)
    bf16_misaligned[4] = ctypes.c_int32(1)
    bf16_misaligned[3] = ctypes.c_int64(12)
    bf16_misaligned[2] = ctypes.c_int32(12)
    assert lib.hme_assign(*bf16_misaligned) == 1 and b"TMA" in lib.hme_last_error()
    for flags in (8, 3):  # an unknown bit; PREPARED together with PREPARE_OUT
        bad_flags = list(args)
        bad_flags[7] = ctypes.c_int32(flags)
        assert lib.hme_assign(*bad_flags) == 1 and b"flags" in lib.hme_last_error()
    lib.hme_partition.restype = ctypes.c_int
    # tag arrays must be all or none
    assert lib.hme_partition(p(16), ctypes.c_int64(4), ctypes.c_int32(2), p(16), p(16), p(16), None, p(16), None,
                             None, None, p(256), ctypes.c_size_t(1 << 20), None) == 1



def test_assign_rows_and_noalloc_partition_host_validation(lib):
    """hme_assign_rows refuses row ranges outside [0, N), bad flags and missing
    outputs, and hme_partition_noalloc refuses sizes outside its limits and
    missing outputs, on the host before any CUDA call (no GPU here)."""
    p, i64, i32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32
    lib.hme_last_error.restype = ctypes.c_char_p
    f = lib.hme_assign_rows
    f.restype = ctypes.c_int
    f.argtypes = [p, i64, i64, i64, i32, i64, i32, p, i32, i32, p, p, p, p, ctypes.c_size_t, p]
    # X, N, row0, row1, d, ldx, dtype, C, K, flags, labels, mind, objective, ws, ws_bytes, stream
    ok = [p(256), 100, 0, 100, 8, 8, 0, p(256), 4, 0, p(256), None, None, p(256), 1 << 30, None]
    cases = [({2: -1}, 1, b"rows"), ({3: 101}, 1, b"rows"), ({2: 60, 3: 50}, 1, b"rows"),
             ({9: 8}, 1, b"flags"), ({7: None}, 1, b"C"), ({10: None}, 1, b"labels_out"),
             ({13: p(257)}, 1, b"aligned"), ({14: 16}, 2, b"")]
    for change, code, word in cases:
        args = list(ok)
        for i, v in change.items():
            args[i] = v
        assert f(*args) == code, change
        assert word in lib.hme_last_error(), change
    g = lib.hme_partition_noalloc
    g.restype = ctypes.c_int
    g.argtypes = [p, i64, i32, p, p, p, p, p, p]
    # labels, N, K, hist, offsets, perm, sorted labels, status, stream
    ok = [p(256), 100, 4, p(256), p(256), p(256), None, None, None]
    for i, bad in [(1, -1), (1, 2**31), (2, 0), (2, 16385), (3, None), (4, None), (0, None), (5, None)]:
        args = list(ok)
        args[i] = bad
        assert g(*args) == 1, (i, bad)  # HME_EINVAL

def test_product_path_has_no_oracle_import():
    """The product package never imports, links or runs the oracle."""
    pkg = os.path.join(ROOT, "paper_1704_06363_gb300")
    for dirpath, _, files in os.walk(pkg):
        for fn in files:
            if fn.endswith((".py", ".cu", ".cuh", ".h")):
                text = open(os.path.join(dirpath, fn)).read()
                assert "import oracle" not in text and "from oracle" not in text and "liboracle" not in text, fn


def test_tag_hist_host_validation(lib):
    f = lib.hme_workspace_bytes
    f.restype = ctypes.c_size_t
    f.argtypes = [ctypes.c_int32, ctypes.c_int64, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32]
    assert f(4, 16_000_000, 20_000, 1024, 0) >= 256 + 1025 * 8  # op 4: d is the vocabulary size
    assert f(4, 10, 0, 4, 0) == 0  # V = 0 rejected
    g = lib.hme_tag_cluster_hist
    g.restype = ctypes.c_int
    p, i64, i32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32
    g.argtypes = [p, p, p, i64, i32, i32, p, p, p, ctypes.c_size_t, p]
    ok = [p(256), p(256), p(256), 10, 4, 100, p(256), None, p(256), 1 << 20, None]
    for i, bad in [(4, 0), (5, 0), (6, None), (0, None), (9, 8)]:  # K = 0, V = 0, no counts, no offsets, tiny ws
        args = list(ok)
        args[i] = bad
        assert g(*args) != 0


def test_pca_host_validation(lib):
    f = lib.hme_workspace_bytes
    f.restype = ctypes.c_size_t
    f.argtypes = [ctypes.c_int32, ctypes.c_int64, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32]
    full = f(6, 1_000_000, 2048, 256, 0)
    assert full >= 2 * 1_000_000 * 2048 * 2  # the transposed bf16 split of the centred rows
    assert 0 < f(6, 0, 2048, 256, 0) < full  # N = 0: transform only
    assert f(6, 100, 16, 17, 0) == 0  # r > d
    assert f(6, 100, 16, 4, 1) == 0  # bf16 features are not taken
    p, i64, i32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32
    g = lib.hme_pca_fit
    g.restype = ctypes.c_int
    g.argtypes = [p, i64, i32, i64, i32, i32, p, p, p, p, p, ctypes.c_size_t, p]
    ok = [p(256), 100, 16, 16, 0, 4, p(256), p(256), None, None, p(256), 1 << 30, None]
    for i, bad in [(1, 0), (4, 1), (5, 0), (5, 17), (3, 8), (6, None), (7, None), (10, None), (10, p(300))]:
        args = list(ok)
        args[i] = bad
        assert g(*args) == 1, (i, bad)  # HME_EINVAL before any CUDA call
    args = list(ok)
    args[11] = 64
    assert g(*args) == 2  # workspace too small
    args = list(ok)
    args[2], args[3], args[5] = 8193, 8193, 4
    assert g(*args) == 1 and b"8192" in lib.hme_last_error()  # the Jacobi takes d <= 8192
    t = lib.hme_pca_transform
    t.restype = ctypes.c_int
    t.argtypes = [p, i64, i32, i64, i32, p, p, i32, p, i64, p, ctypes.c_size_t, p]
    tok = [p(256), 100, 300, 300, 0, p(256), p(256), 16, p(256), 16, p(256), 1 << 30, None]
    for i, bad in [(7, 257), (9, 8), (0, p(260)), (3, 302), (8, None)]:  # r > 256, ldz < r, misaligned X / ldx
        args = list(tok)
        args[i] = bad
        assert t(*args) == 1, (i, bad)
    c = lib.hme_pca_covariance
    c.restype = ctypes.c_int
    c.argtypes = [p, i64, i32, i64, i32, p, p, p, ctypes.c_size_t, p]
    assert c(p(256), 0, 4, 4, 0, p(256), p(256), p(256), 1 << 20, None) == 1  # N = 0
    assert c(p(256), 10, 4, 4, 0, None, p(256), p(256), 1 << 20, None) == 1


def test_binding_refuses_host_tensors_before_calling_the_library():
    """The C ABI takes device pointers; the binding refuses CPU tensors (and, for
    the streamed features, pageable host memory) with HME_EINVAL before any
    call, so that no kernel is handed a host address."""
    import torch

    from paper_1704_06363_gb300 import hme

    X = torch.zeros(8, 4)
    C = torch.zeros(2, 4)
    ws = torch.zeros(1 << 16, dtype=torch.uint8)
    cases = [
        lambda: hme.hme_assign(X, C, torch.zeros(8, dtype=torch.int32), ws),
        lambda: hme.hme_prepare_features(X, 2, ws),
        lambda: hme.hme_route(X, C, torch.zeros(8, dtype=torch.int32), torch.zeros(3, dtype=torch.int64),
                              torch.zeros(8, dtype=torch.int32), ws),
        lambda: hme.hme_partition(torch.zeros(8, dtype=torch.int32), 2, torch.zeros(2, dtype=torch.int64),
                                  torch.zeros(3, dtype=torch.int64), torch.zeros(8, dtype=torch.int32), ws),
        lambda: hme.hme_kmeans_stream(X, 2, 1, 4, C, torch.zeros(8, dtype=torch.int32), torch.zeros(8), ws),
        lambda: hme.hme_pca_covariance(X, torch.zeros(4, dtype=torch.float64),
                                       torch.zeros(4, 4, dtype=torch.float64), ws),
    ]
    for call in cases:
        with pytest.raises(hme.HmeError) as ei:
            call()
        assert ei.value.code == hme.HME_EINVAL
        assert "CUDA tensors" in str(ei.value)


def test_binding_checks_array_types_and_sizes_before_calling_the_library(monkeypatch):
    """Every array argument is checked for its element type, contiguity and
    length before the C entry point is called: a wrong dtype or a short output
    would otherwise let a kernel write past the tensor.  The device check is
    stubbed out (no GPU here) and the library replaced by a recorder, which must
    never be reached."""
    import torch

    from paper_1704_06363_gb300 import hme

    calls = []

    class Recorder:
        def __getattr__(self, name):
            def f(*a):
                calls.append(name)
                return hme.HME_OK
            return f

        def hme_last_error(self):
            return b""

    monkeypatch.setattr(hme, "lib", lambda: Recorder())
    monkeypatch.setattr(hme, "_ptr", lambda t, host_ok=False: None if t is None else 16)
    monkeypatch.setattr(hme, "_stream", lambda stream: None)

    N, d, K = 8, 4, 3
    X = torch.zeros(N, d)
    C = torch.zeros(K, d)
    ws = torch.zeros(256, dtype=torch.uint8)
    i32, i64, f32, f64 = torch.int32, torch.int64, torch.float32, torch.float64

    def z(n, dt):
        return torch.zeros(n, dtype=dt)

    good_part = dict(hist_out=z(K, i64), offsets_out=z(K + 1, i64), perm_out=z(N, i32))
    bad = [
        # hme_assign: labels int64, labels short, mind float64, C float64, C not contiguous
        lambda: hme.hme_assign(X, C, z(N, i64), ws),
        lambda: hme.hme_assign(X, C, z(N - 1, i32), ws),
        lambda: hme.hme_assign(X, C, z(N, i32), ws, mind_out=z(N, f64)),
        lambda: hme.hme_assign(X, C.double(), z(N, i32), ws),
        lambda: hme.hme_assign(X, torch.zeros(d, K).t(), z(N, i32), ws),
        lambda: hme.hme_assign(X, C, z(N, i32), ws, objective_out=z(1, f32)),
        # hme_update_centroids: counts int32, counts short, prev_labels short
        lambda: hme.hme_update_centroids(X, z(N, i32), None, C, ws, counts_out=z(K, i32)),
        lambda: hme.hme_update_centroids(X, z(N, i32), None, C, ws, counts_out=z(K - 1, i64)),
        lambda: hme.hme_update_centroids(X, z(N, i32), None, C, ws, prev_labels=z(N - 2, i32)),
        lambda: hme.hme_update_centroids(X, z(N, i64), None, C, ws),
        # hme_partition: hist int32, offsets of K entries, perm short, labels int64, sorted labels short
        lambda: hme.hme_partition(z(N, i32), K, z(K, i32), z(K + 1, i64), z(N, i32), ws),
        lambda: hme.hme_partition(z(N, i32), K, z(K, i64), z(K, i64), z(N, i32), ws),
        lambda: hme.hme_partition(z(N, i32), K, z(K, i64), z(K + 1, i64), z(N - 1, i32), ws),
        lambda: hme.hme_partition(z(N, i64), K, **good_part, ws=ws),
        lambda: hme.hme_partition(z(N, i32), K, **good_part, ws=ws, sorted_labels_out=z(N - 1, i32)),
        lambda: hme.hme_partition(z(N, i32), K, **good_part, ws=ws, tag_off=z(N + 1, i64), tags=z(20, i32),
                                  tag_off_out=z(N + 1, i64), tags_out=z(19, i32)),
        lambda: hme.hme_partition(z(N, i32), K, **good_part, ws=ws, tag_off=z(N + 1, i64), tags=z(20, i32)),
        # hme_route: expert short, order int64
        lambda: hme.hme_route(X, C, z(N - 1, i32), z(K + 1, i64), z(N, i32), ws),
        lambda: hme.hme_route(X, C, z(N, i32), z(K + 1, i64), z(N, i64), ws),
        # hme_partition_noalloc: hist short, perm int64
        lambda: hme.hme_partition_noalloc(z(N, i32), K, z(K - 1, i64), z(K + 1, i64), z(N, i32)),
        lambda: hme.hme_partition_noalloc(z(N, i32), K, z(K, i64), z(K + 1, i64), z(N, i64)),
        # hme_tag_cluster_hist: counts short
        lambda: hme.hme_tag_cluster_hist(z(K + 1, i64), z(N + 1, i64), z(10, i32), K, 5, z(K * 5 - 1, i64), ws),
        # hme_kmeans_init: C_out with the wrong number of rows
        lambda: hme.hme_kmeans_init(X, K + 1, 0, hme.HME_INIT_KMEANSPP, C, ws),
        # hme_pca_covariance: cov short
        lambda: hme.hme_pca_covariance(X, z(d, f64), torch.zeros(d, d - 1, dtype=f64), ws),
    ]
    for i, call in enumerate(bad):
        with pytest.raises(hme.HmeError) as ei:
            call()
        assert ei.value.code == hme.HME_EINVAL, i
    assert calls == []
    # the same calls with well-formed arguments reach the library
    hme.hme_assign(X, C, z(N, i32), ws, z(N, f32), z(1, f64))
    hme.hme_partition(z(N, i32), K, **good_part, ws=ws, sorted_labels_out=z(N, i32))
    hme.hme_partition_noalloc(z(N, i32), K, z(K, i64), z(K + 1, i64), z(N, i32))
    assert calls == ["hme_assign", "hme_partition", "hme_partition_noalloc"]
