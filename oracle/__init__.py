"""fp64 CPU oracle for the hard-MoE gater (arXiv 1704.06363, Section 2, Eq. 2).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
package.  The product path (``paper_1704_06363_gb300``) never imports it, and it
never imports the product path: the two share no code.

The arithmetic lives in ``oracle.c`` (plain C, fp64, direct sums); this module
only builds it with gcc and marshals numpy arrays through ctypes.  Feature
matrices are numpy ``float32`` arrays, or bf16 given as ``uint16`` bit patterns
(``dtype="bf16"``).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIBDIR = os.path.join(_HERE, "lib")
_LIB = os.path.join(_LIBDIR, "liboracle.so")

F32, BF16 = 0, 1
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile oracle.c into oracle/lib/liboracle.so (gcc, -O2, OpenMP if available).

    -ffp-contract=off keeps every multiply and add separately rounded, so the
    oracle gives the same fp64 values on x86-64 and AArch64.
    """
    os.makedirs(_LIBDIR, exist_ok=True)
    if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
        return _LIB
    base = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fPIC", "-shared", _SRC, "-o", _LIB + ".tmp", "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True, capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(_LIB + ".tmp", _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        p, i64, i32, u64 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_uint64
        lib.orc_splitmix64_at.restype = u64
        lib.orc_splitmix64_at.argtypes = [u64, u64]
        lib.orc_unit.restype = ctypes.c_double
        lib.orc_unit.argtypes = [u64]
        lib.orc_scaled_index.restype = u64
        lib.orc_scaled_index.argtypes = [u64, u64]
        lib.orc_f32_to_bf16_rne.restype = ctypes.c_uint16
        lib.orc_f32_to_bf16_rne.argtypes = [ctypes.c_float]
        lib.orc_bf16_to_f32.restype = ctypes.c_float
        lib.orc_bf16_to_f32.argtypes = [ctypes.c_uint16]
        lib.orc_kmeanspp.restype = i32
        lib.orc_kmeanspp.argtypes = [p, i64, i64, i64, i32, i64, u64, i32, p, p]
        lib.orc_assign.restype = i32
        lib.orc_assign.argtypes = [p, i64, i64, i64, i32, p, i64, p, p, p, p]
        lib.orc_objective.restype = i32
        lib.orc_objective.argtypes = [p, i64, i64, i64, i32, p, i64, p, p]
        lib.orc_update.restype = i32
        lib.orc_update.argtypes = [p, i64, i64, i64, i32, p, p, i64, p, p, p]
        lib.orc_partition.restype = i32
        lib.orc_partition.argtypes = [p, i64, i64, p, p, p, p, p, p, p, p]
        lib.orc_tag_cluster_hist.restype = i32
        lib.orc_tag_cluster_hist.argtypes = [p, i64, i64, p, p, i64, p, p]
        lib.orc_lloyd.restype = i32
        lib.orc_lloyd.argtypes = [p, i64, i64, i64, i32, p, i64, i64, p, p, p, p]
        _lib = lib
        return lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _features(X, dtype):
    """Return (C-contiguous array, N, d, dtype code)."""
    if dtype == "bf16":
        X = np.ascontiguousarray(X, dtype=np.uint16)
        code = BF16
    elif dtype == "f32":
        X = np.ascontiguousarray(X, dtype=np.float32)
        code = F32
    else:
        raise ValueError(f"dtype must be 'f32' or 'bf16', got {dtype!r}")
    if X.ndim != 2:
        raise ValueError("features must be a 2-D (N, d) array")
    return X, X.shape[0], X.shape[1], code


# --- scalar helpers (exposed so the tests can pin them) ---------------------------

def splitmix64_at(seed: int, j: int) -> int:
    return int(_load().orc_splitmix64_at(seed & (2**64 - 1), j & (2**64 - 1)))


def unit(r: int) -> float:
    return float(_load().orc_unit(r))


def scaled_index(r: int, n: int) -> int:
    return int(_load().orc_scaled_index(r, n))


def f32_to_bf16_rne(x: float) -> int:
    return int(_load().orc_f32_to_bf16_rne(x))


def bf16_to_f32(b: int) -> float:
    return float(_load().orc_bf16_to_f32(b))


# --- the method --------------------------------------------------------------------

def kmeanspp(X, K: int, seed: int, subsample: bool = False, dtype: str = "f32"):
    """k-means++ seeding.  Returns (C[K, d] float32, picked rows[K] int64)."""
    X, N, d, code = _features(X, dtype)
    C = np.zeros((K, d), np.float32)
    picked = np.zeros(K, np.int64)
    rc = _load().orc_kmeanspp(_ptr(X), N, d, d, code, K, seed & (2**64 - 1), int(bool(subsample)),
                              _ptr(C), _ptr(picked))
    if rc != 0:
        raise ValueError("orc_kmeanspp: bad arguments")
    return C, picked


def assign(X, C, dtype: str = "f32"):
    """Eq. 2.  Returns (labels int32[N], d1 f64[N], d2 f64[N], objective float)."""
    X, N, d, code = _features(X, dtype)
    C = np.ascontiguousarray(C, np.float32)
    if C.ndim != 2 or C.shape[1] != d:
        raise ValueError("C must be (K, d)")
    K = C.shape[0]
    labels = np.zeros(N, np.int32)
    d1 = np.zeros(N, np.float64)
    d2 = np.zeros(N, np.float64)
    J = ctypes.c_double(0.0)
    if _load().orc_assign(_ptr(X), N, d, d, code, _ptr(C), K, _ptr(labels), _ptr(d1), _ptr(d2), ctypes.byref(J)):
        raise MemoryError("orc_assign: allocation failed")
    return labels, d1, d2, J.value


def objective(X, C, labels, dtype: str = "f32") -> float:
    """J = sum_i ||x_i - c_{labels[i]}||^2 (fp64), centres bf16-rounded for bf16 features."""
    X, N, d, code = _features(X, dtype)
    C = np.ascontiguousarray(C, np.float32)
    labels = np.ascontiguousarray(labels, np.int32)
    J = ctypes.c_double(0.0)
    if _load().orc_objective(_ptr(X), N, d, d, code, _ptr(C), C.shape[0], _ptr(labels), ctypes.byref(J)) != 0:
        raise ValueError("orc_objective: label out of range")
    return J.value


def update(X, labels, mind, C, dtype: str = "f32"):
    """Centre step + empty-cluster reseed.  Returns (C_new f32[K,d], counts i64[K], n_reseeded)."""
    X, N, d, code = _features(X, dtype)
    C = np.array(C, np.float32, order="C", copy=True)
    K = C.shape[0]
    labels = np.ascontiguousarray(labels, np.int32)
    mind = None if mind is None else np.ascontiguousarray(mind, np.float64)
    counts = np.zeros(K, np.int64)
    nr = ctypes.c_int32(0)
    rc = _load().orc_update(_ptr(X), N, d, d, code, _ptr(labels), _ptr(mind), K, _ptr(C), _ptr(counts),
                            ctypes.byref(nr))
    if rc != 0:
        raise ValueError("orc_update: label out of range")
    return C, counts, nr.value


def partition(labels, K: int, tag_off=None, tags=None):
    """Stable counting sort by expert.  Returns dict(hist, offsets, perm, sorted_labels[, tag_off, tags])."""
    labels = np.ascontiguousarray(labels, np.int32)
    N = labels.shape[0]
    hist = np.zeros(K, np.int64)
    offsets = np.zeros(K + 1, np.int64)
    perm = np.zeros(N, np.int32)
    sl = np.zeros(N, np.int32)
    out = dict(hist=hist, offsets=offsets, perm=perm, sorted_labels=sl)
    to = tg = too = tgo = None
    if tag_off is not None:
        to = np.ascontiguousarray(tag_off, np.int64)
        tg = np.ascontiguousarray(tags, np.int32)
        too = np.zeros(N + 1, np.int64)
        tgo = np.zeros(max(1, tg.shape[0]), np.int32)
    rc = _load().orc_partition(_ptr(labels), N, K, _ptr(hist), _ptr(offsets), _ptr(perm), _ptr(sl),
                               _ptr(to), _ptr(tg), _ptr(too), _ptr(tgo))
    if rc != 0:
        raise ValueError("orc_partition: label out of range")
    if tag_off is not None:
        out["tag_off"] = too
        out["tags"] = tgo[: tg.shape[0]]
    return out


def tag_cluster_hist(labels, K: int, tag_off, tags, V: int):
    """Section 4.5 tag statistics of a clustering: (counts i64[K, V], sparsity f64[V]).

    counts[k, t] = occurrences of tag t among the tags of the points in cluster k;
    sparsity[t] = ||counts[:, t]||_1 / ||counts[:, t]||_2, 0 for an absent tag.
    """
    labels = np.ascontiguousarray(labels, np.int32)
    N = labels.shape[0]
    to = np.ascontiguousarray(tag_off, np.int64)
    tg = np.ascontiguousarray(tags, np.int32)
    if tg.shape[0] == 0:
        tg = np.zeros(1, np.int32)
    counts = np.zeros((K, V), np.int64)
    sp = np.zeros(V, np.float64)
    rc = _load().orc_tag_cluster_hist(_ptr(labels), N, K, _ptr(to), _ptr(tg), V, _ptr(counts), _ptr(sp))
    if rc != 0:
        raise ValueError("orc_tag_cluster_hist: label or tag out of range")
    return counts, sp


def lloyd(X, C0, T: int, dtype: str = "f32"):
    """T free-running Lloyd iterations from C0.

    Returns (C_T f32[K,d], labels of the last assign, objectives f64[T],
    changed i64[T], counts of the last update i64[K]).
    """
    X, N, d, code = _features(X, dtype)
    C = np.array(C0, np.float32, order="C", copy=True)
    K = C.shape[0]
    labels = np.zeros(N, np.int32)
    objs = np.zeros(max(T, 1), np.float64)
    changed = np.zeros(max(T, 1), np.int64)
    counts = np.zeros(K, np.int64)
    rc = _load().orc_lloyd(_ptr(X), N, d, d, code, _ptr(C), K, T, _ptr(labels), _ptr(objs), _ptr(changed),
                           _ptr(counts))
    if rc != 0:
        raise ValueError("orc_lloyd failed")
    return C, labels, objs[:T], changed[:T], counts


def route(Q, C, dtype: str = "f32"):
    """Eq. 2 on a new batch, then the expert partition of its labels."""
    labels, d1, d2, _ = assign(Q, C, dtype)
    part = partition(labels, C.shape[0])
    return labels, part
