"""ctypes binding of libhme (include/hme.h): argument marshalling only.

Every function takes torch tensors that live on the current CUDA device,
passes their data pointers and sizes to the C entry point of the same name,
and raises ``HmeError`` on a non-zero status.  All arithmetic runs in the CUDA
kernels of ``csrc/``; there is no CPU fallback: if ``lib/libhme.so`` has not
been built (``paper_1704_06363_gb300._build.build()``), importing the library
fails loudly.
"""
from __future__ import annotations

import ctypes
import os
import threading
from typing import Optional

import torch

HME_OK, HME_EINVAL, HME_ENOMEM, HME_ECUDA, HME_ETIMEOUT, HME_EINTERNAL = range(6)
HME_F32, HME_BF16 = 0, 1
HME_OP_INIT, HME_OP_ASSIGN, HME_OP_PARTITION, HME_OP_ROUTE, HME_OP_TAG_HIST, HME_OP_STREAM, HME_OP_PCA = range(7)
HME_INIT_KMEANSPP, HME_INIT_KMEANSPP_SUBSAMPLE = 0, 1
HME_ASSIGN_DEFAULT, HME_ASSIGN_PREPARED, HME_ASSIGN_PREPARE_OUT, HME_ASSIGN_TF32 = 0, 1, 2, 4

_NAMES = {0: "HME_OK", 1: "HME_EINVAL", 2: "HME_ENOMEM", 3: "HME_ECUDA", 4: "HME_ETIMEOUT", 5: "HME_EINTERNAL"}
LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "lib", "libhme.so")

_lock = threading.Lock()
_lib = None


class HmeError(RuntimeError):
    def __init__(self, code: int, fn: str, msg: str):
        super().__init__(f"{fn}: {_NAMES.get(code, code)}: {msg}")
        self.code = code


def lib():
    """The loaded libhme (built in-tree).  Raises if it is missing."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"libhme is not built ({LIB_PATH} missing): run paper_1704_06363_gb300._build.build()")
        L = ctypes.CDLL(LIB_PATH)
        p, i64, i32, u64, sz = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_uint64, ctypes.c_size_t
        L.hme_workspace_bytes.restype = sz
        L.hme_workspace_bytes.argtypes = [i32, i64, i32, i32, i32]
        L.hme_last_error.restype = ctypes.c_char_p
        L.hme_last_error.argtypes = []
        L.hme_sync_status.restype = ctypes.c_int
        L.hme_sync_status.argtypes = [p, p]
        L.hme_kmeans_init.restype = ctypes.c_int
        L.hme_kmeans_init.argtypes = [p, i64, i32, i64, i32, i32, u64, i32, p, p, sz, p]
        L.hme_prepare_features.restype = ctypes.c_int
        L.hme_prepare_features.argtypes = [p, i64, i32, i64, i32, i32, p, sz, p]
        L.hme_assign.restype = ctypes.c_int
        L.hme_assign.argtypes = [p, i64, i32, i64, i32, p, i32, i32, p, p, p, p, sz, p]
        L.hme_assign_rows.restype = ctypes.c_int
        L.hme_assign_rows.argtypes = [p, i64, i64, i64, i32, i64, i32, p, i32, i32, p, p, p, p, sz, p]
        L.hme_update_centroids.restype = ctypes.c_int
        L.hme_update_centroids.argtypes = [p, i64, i32, i64, i32, p, p, p, i32, p, p, p, p, p, sz, p]
        L.hme_partition.restype = ctypes.c_int
        L.hme_partition.argtypes = [p, i64, i32, p, p, p, p, p, p, p, p, p, sz, p]
        L.hme_route.restype = ctypes.c_int
        L.hme_route.argtypes = [p, i64, i32, i64, i32, p, i32, i32, p, p, p, p, sz, p]
        L.hme_partition_noalloc.restype = ctypes.c_int
        L.hme_partition_noalloc.argtypes = [p, i64, i32, p, p, p, p, p, p]
        L.hme_kmeans_stream.restype = ctypes.c_int
        L.hme_kmeans_stream.argtypes = [p, i64, i32, i64, i32, i32, i32, i64, p, p, p, p, p, p, p, sz, p]
        L.hme_tag_cluster_hist.restype = ctypes.c_int
        L.hme_tag_cluster_hist.argtypes = [p, p, p, i64, i32, i32, p, p, p, sz, p]
        L.hme_pca_covariance.restype = ctypes.c_int
        L.hme_pca_covariance.argtypes = [p, i64, i32, i64, i32, p, p, p, sz, p]
        L.hme_pca_fit.restype = ctypes.c_int
        L.hme_pca_fit.argtypes = [p, i64, i32, i64, i32, i32, p, p, p, p, p, sz, p]
        L.hme_pca_transform.restype = ctypes.c_int
        L.hme_pca_transform.argtypes = [p, i64, i32, i64, i32, p, p, i32, p, i64, p, sz, p]
        L.hme_launch_count.restype = i64
        L.hme_launch_count.argtypes = []
        L.hme_debug_bounded_wait.restype = ctypes.c_int
        L.hme_debug_bounded_wait.argtypes = [u64, p, sz, p]
        _lib = L
        return L


def _check(rc: int, fn: str):
    if rc != HME_OK:
        raise HmeError(rc, fn, lib().hme_last_error().decode(errors="replace"))


def _ptr(t: Optional[torch.Tensor], host_ok: bool = False):
    """The tensor's address for the C ABI, which takes device pointers on the
    current CUDA device (hme_kmeans_stream's features may also be page-locked
    host memory).  Anything else would reach a kernel as an address it cannot
    read, so it is refused here, before any call into the library."""
    if t is None:
        return None
    if t.is_cuda:
        cur = torch.cuda.current_device()
        if t.device.index != cur:
            raise HmeError(HME_EINVAL, "argument check",
                           f"a tensor on {t.device} was passed while the current CUDA device is cuda:{cur}; "
                           "the library runs on the current device")
    elif not (host_ok and t.is_pinned()):
        raise HmeError(HME_EINVAL, "argument check",
                       "arguments must be CUDA tensors (device memory)"
                       + (" or, for the features, page-locked host tensors" if host_ok else "")
                       + f"; got a tensor on {t.device}")
    return ctypes.c_void_p(t.data_ptr())


def _arg(t: Optional[torch.Tensor], name: str, dtype: torch.dtype, numel: int, host_ok: bool = False):
    """The address of an array argument after checking what the kernels assume
    of it: element type `dtype`, contiguous, at least `numel` elements (the
    kernels read or write that many), on the current device.  A mismatch would
    let a kernel write past the tensor or misread it, so it is refused with
    HME_EINVAL before any call into the library.  None passes through (the C
    ABI's NULL)."""
    if t is None:
        return None
    if t.dtype != dtype:
        raise HmeError(HME_EINVAL, "argument check", f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise HmeError(HME_EINVAL, "argument check", f"{name} must be contiguous")
    if t.numel() < numel:
        raise HmeError(HME_EINVAL, "argument check",
                       f"{name} has {t.numel()} elements; the call needs at least {numel}")
    return _ptr(t, host_ok)


def _labels(t: torch.Tensor, name: str = "labels") -> int:
    """N of a label vector: a 1-D int32 tensor."""
    if t.dim() != 1:
        raise HmeError(HME_EINVAL, "argument check", f"{name} must be 1-D, got shape {tuple(t.shape)}")
    return t.shape[0]


def _centres(C: torch.Tensor, d: int, name: str = "C") -> int:
    """K of a centre matrix: K x d float32, contiguous."""
    if C.dim() != 2 or C.shape[1] != d:
        raise HmeError(HME_EINVAL, "argument check", f"{name} must be K x {d}, got shape {tuple(C.shape)}")
    return C.shape[0]


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _features(X: torch.Tensor):
    if X.dim() != 2 or X.stride(1) != 1:
        raise ValueError("features must be a 2-D tensor with unit column stride")
    if X.dtype == torch.float32:
        dt = HME_F32
    elif X.dtype == torch.bfloat16:
        dt = HME_BF16
    else:
        raise TypeError(f"features must be float32 or bfloat16, got {X.dtype}")
    return X.shape[0], X.shape[1], max(X.stride(0), X.shape[1]), dt


def _ws(ws: torch.Tensor):
    if not ws.is_contiguous():
        raise HmeError(HME_EINVAL, "argument check", "the workspace must be contiguous")
    return _ptr(ws), ws.numel() * ws.element_size()


def hme_workspace_bytes(op: int, N: int, d: int, K: int, dtype: int) -> int:
    return int(lib().hme_workspace_bytes(op, N, d, K, dtype))


def workspace(op: int, N: int, d: int, K: int, dtype: int, device=None) -> torch.Tensor:
    """A device byte tensor large enough for `op` (torch allocations are 512-byte aligned)."""
    n = hme_workspace_bytes(op, N, d, K, dtype)
    if n == 0:
        raise HmeError(HME_EINVAL, "hme_workspace_bytes", lib().hme_last_error().decode(errors="replace"))
    return torch.empty(n, dtype=torch.uint8, device=device if device is not None else "cuda")


def hme_sync_status(ws: torch.Tensor, stream=None) -> int:
    """Wait for the stream and return the device-side status of the last call on ws (no raise)."""
    return int(lib().hme_sync_status(_ptr(ws), _stream(stream)))


def hme_last_error() -> str:
    """The message of the last failed call on this thread."""
    return lib().hme_last_error().decode(errors="replace")


def hme_kmeans_init(X: torch.Tensor, K: int, seed: int, method: int, C_out: torch.Tensor, ws: torch.Tensor,
                    stream=None):
    N, d, ldx, dt = _features(X)
    if _centres(C_out, d, "C_out") != K:
        raise HmeError(HME_EINVAL, "argument check", f"C_out must have K = {K} rows")
    w, wb = _ws(ws)
    _check(lib().hme_kmeans_init(_ptr(X), N, d, ldx, dt, K, seed & (2**64 - 1), method,
                                 _arg(C_out, "C_out", torch.float32, K * d), w, wb,
                                 _stream(stream)), "hme_kmeans_init")


def hme_prepare_features(X: torch.Tensor, K: int, ws: torch.Tensor, stream=None):
    N, d, ldx, dt = _features(X)
    w, wb = _ws(ws)
    _check(lib().hme_prepare_features(_ptr(X), N, d, ldx, dt, K, w, wb, _stream(stream)), "hme_prepare_features")


def hme_assign(X: torch.Tensor, C: torch.Tensor, labels_out: torch.Tensor, ws: torch.Tensor,
               mind_out: Optional[torch.Tensor] = None, objective_out: Optional[torch.Tensor] = None,
               flags: int = HME_ASSIGN_DEFAULT, stream=None):
    N, d, ldx, dt = _features(X)
    K = _centres(C, d)
    w, wb = _ws(ws)
    _check(lib().hme_assign(_ptr(X), N, d, ldx, dt, _arg(C, "C", torch.float32, K * d), K, flags,
                            _arg(labels_out, "labels_out", torch.int32, N),
                            _arg(mind_out, "mind_out", torch.float32, N),
                            _arg(objective_out, "objective_out", torch.float64, 1), w, wb, _stream(stream)),
           "hme_assign")


def hme_assign_rows(X: torch.Tensor, row0: int, row1: int, C: torch.Tensor, labels_out: torch.Tensor,
                    ws: torch.Tensor, mind_out: Optional[torch.Tensor] = None,
                    objective_out: Optional[torch.Tensor] = None, flags: int = HME_ASSIGN_DEFAULT, stream=None):
    """hme_assign of rows [row0, row1) of X (all N rows' workspace and outputs)."""
    N, d, ldx, dt = _features(X)
    K = _centres(C, d)
    w, wb = _ws(ws)
    _check(lib().hme_assign_rows(_ptr(X), N, row0, row1, d, ldx, dt, _arg(C, "C", torch.float32, K * d), K, flags,
                                 _arg(labels_out, "labels_out", torch.int32, N),
                                 _arg(mind_out, "mind_out", torch.float32, N),
                                 _arg(objective_out, "objective_out", torch.float64, 1), w, wb, _stream(stream)),
           "hme_assign_rows")


def hme_update_centroids(X: torch.Tensor, labels: torch.Tensor, mind: Optional[torch.Tensor], C_inout: torch.Tensor,
                         ws: torch.Tensor, counts_out: Optional[torch.Tensor] = None,
                         n_reseeded_out: Optional[torch.Tensor] = None, objective_out: Optional[torch.Tensor] = None,
                         prev_labels: Optional[torch.Tensor] = None, stream=None):
    """Centre step.  prev_labels: the labels of the previous call on this ws (incremental update)."""
    N, d, ldx, dt = _features(X)
    K = _centres(C_inout, d, "C_inout")
    w, wb = _ws(ws)
    _check(lib().hme_update_centroids(_ptr(X), N, d, ldx, dt, _arg(labels, "labels", torch.int32, N),
                                      _arg(prev_labels, "prev_labels", torch.int32, N),
                                      _arg(mind, "mind", torch.float32, N), K,
                                      _arg(C_inout, "C_inout", torch.float32, K * d),
                                      _arg(counts_out, "counts_out", torch.int64, K),
                                      _arg(n_reseeded_out, "n_reseeded_out", torch.int32, 1),
                                      _arg(objective_out, "objective_out", torch.float64, 1), w, wb,
                                      _stream(stream)),
           "hme_update_centroids")


def hme_partition(labels: torch.Tensor, K: int, hist_out: torch.Tensor, offsets_out: torch.Tensor,
                  perm_out: torch.Tensor, ws: torch.Tensor, sorted_labels_out: Optional[torch.Tensor] = None,
                  tag_off: Optional[torch.Tensor] = None, tags: Optional[torch.Tensor] = None,
                  tag_off_out: Optional[torch.Tensor] = None, tags_out: Optional[torch.Tensor] = None, stream=None):
    N = _labels(labels)
    lists = [t is None for t in (tag_off, tags, tag_off_out, tags_out)]
    if any(lists) and not all(lists):
        raise HmeError(HME_EINVAL, "argument check", "tag_off, tags, tag_off_out and tags_out: all four or none")
    T = tags.numel() if tags is not None else 0
    w, wb = _ws(ws)
    _check(lib().hme_partition(_arg(labels, "labels", torch.int32, N), N, K,
                               _arg(hist_out, "hist_out", torch.int64, K),
                               _arg(offsets_out, "offsets_out", torch.int64, K + 1),
                               _arg(perm_out, "perm_out", torch.int32, N),
                               _arg(sorted_labels_out, "sorted_labels_out", torch.int32, N),
                               _arg(tag_off, "tag_off", torch.int64, N + 1), _arg(tags, "tags", torch.int32, 0),
                               _arg(tag_off_out, "tag_off_out", torch.int64, N + 1),
                               _arg(tags_out, "tags_out", torch.int32, T),
                               w, wb, _stream(stream)), "hme_partition")


def hme_route(Q: torch.Tensor, C: torch.Tensor, expert_out: torch.Tensor, offsets_out: torch.Tensor,
              order_out: torch.Tensor, ws: torch.Tensor, flags: int = HME_ASSIGN_DEFAULT, stream=None):
    B, d, ldq, dt = _features(Q)
    K = _centres(C, d)
    w, wb = _ws(ws)
    _check(lib().hme_route(_ptr(Q), B, d, ldq, dt, _arg(C, "C", torch.float32, K * d), K, flags,
                           _arg(expert_out, "expert_out", torch.int32, B),
                           _arg(offsets_out, "offsets_out", torch.int64, K + 1),
                           _arg(order_out, "order_out", torch.int32, B), w, wb, _stream(stream)), "hme_route")


def hme_kmeans_stream(X: torch.Tensor, K: int, iters: int, chunk_rows: int, C_inout: torch.Tensor,
                      labels_out: torch.Tensor, mind_out: torch.Tensor, ws: torch.Tensor,
                      objectives_out: Optional[torch.Tensor] = None, counts_out: Optional[torch.Tensor] = None,
                      n_reseeded_out: Optional[torch.Tensor] = None, stream=None):
    """Lloyd's iterations on X in page-locked host memory (or device memory), streamed in chunks."""
    N, d, ldx, dt = _features(X)
    if _centres(C_inout, d, "C_inout") != K:
        raise HmeError(HME_EINVAL, "argument check", f"C_inout must have K = {K} rows")
    w, wb = _ws(ws)
    _check(lib().hme_kmeans_stream(_ptr(X, host_ok=True), N, d, ldx, dt, K, iters, chunk_rows,
                                   _arg(C_inout, "C_inout", torch.float32, K * d),
                                   _arg(labels_out, "labels_out", torch.int32, N),
                                   _arg(mind_out, "mind_out", torch.float32, N),
                                   _arg(objectives_out, "objectives_out", torch.float64, max(iters, 0)),
                                   _arg(counts_out, "counts_out", torch.int64, K),
                                   _arg(n_reseeded_out, "n_reseeded_out", torch.int32, 1), w,
                                   wb, _stream(stream)), "hme_kmeans_stream")


def hme_tag_cluster_hist(offsets: torch.Tensor, tag_off: torch.Tensor, tags: torch.Tensor, K: int, V: int,
                         counts_out: torch.Tensor, ws: torch.Tensor, sparsity_out: Optional[torch.Tensor] = None,
                         stream=None):
    """Section 4.5 tag statistics from hme_partition's outputs: counts_out[K, V] int64, sparsity_out[V] fp64."""
    N = _labels(tag_off, "tag_off") - 1
    w, wb = _ws(ws)
    _check(lib().hme_tag_cluster_hist(_arg(offsets, "offsets", torch.int64, K + 1),
                                      _arg(tag_off, "tag_off", torch.int64, N + 1), _arg(tags, "tags", torch.int32, 0),
                                      N, K, V, _arg(counts_out, "counts_out", torch.int64, K * V),
                                      _arg(sparsity_out, "sparsity_out", torch.float64, V), w, wb, _stream(stream)),
           "hme_tag_cluster_hist")


def hme_pca_covariance(X: torch.Tensor, mean_out: torch.Tensor, cov_out: torch.Tensor, ws: torch.Tensor,
                       stream=None):
    """Section 4.2 PCA: column mean (fp64, d) and covariance (fp64, d x d) of fp32 features."""
    N, d, ldx, dt = _features(X)
    w, wb = _ws(ws)
    _check(lib().hme_pca_covariance(_ptr(X), N, d, ldx, dt, _arg(mean_out, "mean_out", torch.float64, d),
                                    _arg(cov_out, "cov_out", torch.float64, d * d), w, wb, _stream(stream)),
           "hme_pca_covariance")


def hme_pca_fit(X: torch.Tensor, r: int, mean_out: torch.Tensor, components_out: torch.Tensor, ws: torch.Tensor,
                variances_out: Optional[torch.Tensor] = None, stream=None) -> int:
    """Section 4.2 PCA: mean (fp32, d), r leading components (fp32, r x d) and their variances; returns the
    Jacobi sweeps made (the call synchronises the stream once per sweep)."""
    N, d, ldx, dt = _features(X)
    w, wb = _ws(ws)
    sweeps = ctypes.c_int32(0)
    _check(lib().hme_pca_fit(_ptr(X), N, d, ldx, dt, r, _arg(mean_out, "mean_out", torch.float32, d),
                             _arg(components_out, "components_out", torch.float32, r * d),
                             _arg(variances_out, "variances_out", torch.float32, r),
                             ctypes.byref(sweeps), w, wb, _stream(stream)), "hme_pca_fit")
    return int(sweeps.value)


def hme_pca_transform(X: torch.Tensor, mean: torch.Tensor, components: torch.Tensor, Z_out: torch.Tensor,
                      ws: torch.Tensor, stream=None):
    """Z_out[i, j] = components[j] . (x_i - mean), fp32 (N x r)."""
    N, d, ldx, dt = _features(X)
    r = _centres(components, d, "components")
    if Z_out.dim() != 2 or Z_out.stride(1) != 1:
        raise ValueError("Z_out must be a 2-D tensor with unit column stride")
    if Z_out.dtype != torch.float32 or Z_out.shape[0] < N or Z_out.shape[1] < r:
        raise HmeError(HME_EINVAL, "argument check",
                       f"Z_out must be float32 with at least {N} x {r} elements, got {Z_out.dtype} {tuple(Z_out.shape)}")
    w, wb = _ws(ws)
    _check(lib().hme_pca_transform(_ptr(X), N, d, ldx, dt, _arg(mean, "mean", torch.float32, d),
                                   _arg(components, "components", torch.float32, r * d), r, _ptr(Z_out),
                                   max(Z_out.stride(0), r), w, wb, _stream(stream)), "hme_pca_transform")


def hme_partition_noalloc(labels: torch.Tensor, K: int, hist_out: torch.Tensor, offsets_out: torch.Tensor,
                          perm_out: torch.Tensor, sorted_labels_out: Optional[torch.Tensor] = None,
                          status_out: Optional[torch.Tensor] = None, stream=None):
    """hme_partition without a workspace (for callers that cannot allocate device memory)."""
    N = _labels(labels)
    _check(lib().hme_partition_noalloc(_arg(labels, "labels", torch.int32, N), N, K,
                                       _arg(hist_out, "hist_out", torch.int64, K),
                                       _arg(offsets_out, "offsets_out", torch.int64, K + 1),
                                       _arg(perm_out, "perm_out", torch.int32, N),
                                       _arg(sorted_labels_out, "sorted_labels_out", torch.int32, N),
                                       _arg(status_out, "status_out", torch.int32, 1), _stream(stream)),
           "hme_partition_noalloc")


def hme_launch_count() -> int:
    return int(lib().hme_launch_count())


def hme_debug_bounded_wait(timeout_ns: int, ws: torch.Tensor, stream=None):
    w, wb = _ws(ws)
    _check(lib().hme_debug_bounded_wait(timeout_ns, w, wb, _stream(stream)), "hme_debug_bounded_wait")
