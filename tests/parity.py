"""Tolerance checks shared by the GPU parity tests.

The oracle (fp64, direct sums) is the reference; the bars are:
  - assignments: a GPU label may differ from the oracle's only where the
    oracle's top-2 gap (D2 - D1) / D2 is below 1e-4, and then the GPU's choice
    must itself be within 1e-4 * D2 of the best distance;
  - distances from hme_assign (norm expansion on the tensor cores): within
    ceil(d/16) * nprod * 2^-23 (||x||^2 + ||c||^2)  [one ulp of the fp32
    accumulator per accumulation step, the observed accumulation rounds
    towards zero]  + 2^-15 (||x|| + ||c||) ||x - c||  [fp32 features: the
    16-bit split, |x - x_eff| <= 2^-16 |x| per element]  + 2^-14 ||x|| ||c||
    [fp32 features: the product xl.cl of the split is not formed,
    2 |xl.cl| <= 2^-15 (1 + 2^-8)^2 ||x|| ||c||]  + 1e-5 D; fp32 features
    assigned with HME_ASSIGN_TF32 (K > 256) are multiplied as tf32 operands
    (10-bit significands: |x - x'| <= 2^-10 |x|, |c - c'| <= 2^-11 |c|),
    whose distances are within ceil(d/8) 2^-23 (||x||^2 + ||c||^2) + 3.001
    2^-10 ||x|| ||c|| (2 |x.c - x'.c'|) + 2^-15 ||x||^2 (norms taken from the
    split of a preparation) + 1e-5 D; the sum of those distances
    (hme_assign's objective estimate) within the sum of the per-row bounds +
    1e-5 J;
  - objective of hme_update_centroids (direct differences): within 1e-5
    relative of the fp64 value for the same (C, labels);
  - centres: ||dc_k||_inf <= 1e-4 * max(||c_k||_inf, 1e-6 max_k ||c_k||_inf);
  - partitions, histograms, counts: bit-exact.
"""
from __future__ import annotations

import numpy as np

import oracle

ASSIGN_GAP = 1e-4
OBJ_RTOL = 1e-5
CENTRE_RTOL = 1e-4


def centre_values(C: np.ndarray, dtype: str) -> np.ndarray:
    """The centres the assign step compares against (bf16-rounded for bf16 features), as fp64."""
    if dtype == "bf16":
        b = np.array([oracle.f32_to_bf16_rne(float(v)) for v in C.ravel()], np.uint16)
        return (b.astype(np.uint32) << 16).view(np.float32).reshape(C.shape).astype(np.float64)
    return C.astype(np.float64)


def features_f64(Xh: np.ndarray, dtype: str) -> np.ndarray:
    if dtype == "bf16":
        return (Xh.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return Xh.astype(np.float64)


def distance_bound(Xd, Cd, labels, D, dtype, tf32=False):
    """Per-row bound on |D_gpu - D| for hme_assign's distances (see the module docstring)."""
    d = Xd.shape[1]
    nprod = 3 if dtype == "f32" else 1
    xn = (Xd ** 2).sum(1)
    cn = (Cd ** 2).sum(1)[labels]
    if dtype == "f32" and tf32:
        return (np.ceil(d / 8) * 2.0 ** -23 * (xn + cn) + 3.001 * 2.0 ** -10 * np.sqrt(xn) * np.sqrt(cn)
                + 2.0 ** -15 * xn + 1e-5 * D)
    b = np.ceil(d / 16) * nprod * 2.0 ** -23 * (xn + cn) + 1e-5 * D
    if dtype == "f32":
        b += 2.0 ** -15 * (np.sqrt(xn) + np.sqrt(cn)) * np.sqrt(np.maximum(D, 0))
        b += 2.0 ** -14 * np.sqrt(xn) * np.sqrt(cn)
    return b


def rel_gap(d1, d2):
    """The oracle's top-2 gap (D2 - D1) / D2 per row; +inf where there is no
    runner-up (K = 1: D2 = inf), so such rows are never near ties."""
    d1 = np.asarray(d1, np.float64)
    d2 = np.asarray(d2, np.float64)
    gap = np.full(d1.shape, np.inf)
    fin = np.isfinite(d2)
    gap[fin] = (d2[fin] - d1[fin]) / np.maximum(d2[fin], 1e-30)
    return gap


def check_assign(Xh, dtype, C, labels, mind=None, objective=None, ref=None, tf32=False):
    """Compare a GPU assignment with the oracle's on the same (X, C).  Returns stats."""
    lab_ref, d1, d2, J = ref if ref is not None else oracle.assign(Xh, C, dtype)
    labels = np.asarray(labels)
    N = labels.shape[0]
    assert labels.min(initial=0) >= 0 and labels.max(initial=0) < C.shape[0]
    gap = rel_gap(d1, d2)
    bad = np.nonzero(labels != lab_ref)[0]
    assert np.all(gap[bad] < ASSIGN_GAP), (
        f"{bad.size} label mismatches, {(gap[bad] >= ASSIGN_GAP).sum()} outside near ties; "
        f"first rows {bad[:8].tolist()}, gaps {gap[bad][:8].tolist()}")
    Xd = features_f64(Xh, dtype)
    Cd = centre_values(C, dtype)
    D_gpu_label = d1.copy()
    if bad.size:
        D_gpu_label[bad] = ((Xd[bad] - Cd[labels[bad]]) ** 2).sum(1)
        assert np.all(D_gpu_label[bad] - d1[bad] <= ASSIGN_GAP * d2[bad])
    bound = distance_bound(Xd, Cd, labels, D_gpu_label, dtype, tf32)
    if mind is not None:
        err = np.abs(np.asarray(mind, np.float64) - D_gpu_label)
        assert np.all(err <= bound + 1e-30), f"distance error up to {np.max(err / (bound + 1e-30)):.3g} x bound"
    if objective is not None:
        Jg = float(D_gpu_label.sum())
        assert abs(float(objective) - Jg) <= OBJ_RTOL * Jg + float(bound.sum()), (float(objective), Jg)
    return dict(N=N, mismatches=int(bad.size), near_ties=int((gap < ASSIGN_GAP).sum()))


def check_objective(J_gpu: float, Xh, dtype, C, labels):
    """hme_update_centroids' objective vs the oracle's J for the same (C, labels): 1e-5 relative."""
    J = oracle.objective(Xh, C, labels, dtype)
    assert abs(float(J_gpu) - J) <= OBJ_RTOL * max(J, 1e-300), (float(J_gpu), J)
    return J


def check_centres(Cg: np.ndarray, Cref: np.ndarray):
    Cg = np.asarray(Cg, np.float64)
    Cref = np.asarray(Cref, np.float64)
    rowmax = np.abs(Cref).max(1)
    scale = np.maximum(rowmax, 1e-6 * rowmax.max())
    err = np.abs(Cg - Cref).max(1)
    worst = int(np.argmax(err / scale))
    assert np.all(err <= CENTRE_RTOL * scale), (
        f"centre {worst}: error {err[worst]:.3g} vs scale {scale[worst]:.3g}")
    return float((err / scale).max())


def check_partition(out_gpu: dict, labels: np.ndarray, K: int, tag_off=None, tags=None):
    ref = oracle.partition(labels, K, tag_off, tags)
    for key in ("hist", "offsets", "perm", "sorted_labels", "tag_off", "tags"):
        if key in out_gpu and out_gpu[key] is not None and key in ref:
            assert np.array_equal(np.asarray(out_gpu[key]), ref[key]), f"{key} differs from the oracle"
    return ref
