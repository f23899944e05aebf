"""Pins for the fp64 CPU oracle, independent of the oracle's own code.

Each test checks the oracle against something the paper or mathematics fixes:
published generator values, hand-computed examples, brute-force optima, the
exact 1-D optimum by dynamic programming (Wang & Song 2011), closed forms,
invariants of Lloyd's iteration, and library routines (numpy's stable argsort,
torch's bf16 rounding, scipy's chi-square test).  Together they are chosen so
that a dropped term, a wrong sign or index, or a swapped operand in the oracle
fails at least one of them.
"""
import itertools
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest
import torch

import oracle
import hme_synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ----------------------------------------------------------------------------------
# random numbers and bf16
# ----------------------------------------------------------------------------------

def test_splitmix64_published_vector():
    vals = [int(l, 16) for l in open(os.path.join(GOLDEN, "splitmix64_seed0.txt")) if l.startswith("0x")]
    assert [oracle.splitmix64_at(0, j) for j in range(len(vals))] == vals


def test_unit_and_scaled_index_exact():
    rng = np.random.RandomState(1)
    for r in [0, 1, 2**11 - 1, 2**11, 2**64 - 1] + [int(v) for v in rng.randint(0, 2**63, 200, dtype=np.int64)]:
        u = oracle.unit(r)
        assert u == float(Fraction(r >> 11, 2**53))
        assert 0.0 <= u < 1.0
        for n in [1, 2, 3, 10_000, 50_000_000, 2**40 + 7]:
            k = oracle.scaled_index(r, n)
            assert k == math.floor(Fraction(r >> 11, 2**53) * n)
            assert 0 <= k < n


def test_bf16_rounding_matches_torch():
    rng = np.random.RandomState(2)
    vals = np.concatenate([
        rng.randn(20000).astype(np.float32) * np.float32(10.0) ** rng.randint(-30, 30, 20000).astype(np.float32),
        np.array([0.0, -0.0, 1.0, 1.00390625, 1.01171875, 3.4e38, -3.4e38, np.inf, -np.inf, 1e-40, -1e-42],
                 np.float32),
        # exact ties between two bf16 values: round to even
        (np.arange(1, 2000, dtype=np.uint32) << 16 | 0x8000).view(np.float32),
    ])
    vals = vals[np.isfinite(vals) | np.isinf(vals)]
    ref = torch.from_numpy(vals).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = np.array([oracle.f32_to_bf16_rne(float(v)) for v in vals], np.uint16)
    assert np.array_equal(got, ref)
    back = np.array([oracle.bf16_to_f32(int(b)) for b in ref[:500]], np.float32)
    assert np.array_equal(back, torch.from_numpy(ref[:500].view(np.int16)).view(torch.bfloat16).float().numpy())


# ----------------------------------------------------------------------------------
# hand-computed examples (Eq. 2 and the centre step)
# ----------------------------------------------------------------------------------

@pytest.mark.parametrize("case", json.load(open(os.path.join(GOLDEN, "kmeans_hand_examples.json")))["cases"],
                         ids=lambda c: c["name"])
def test_hand_examples(case):
    X = np.array(case["X"], np.float32)
    C0 = np.array(case["C0"], np.float32)
    labels, d1, d2, J = oracle.assign(X, C0)
    assert labels.tolist() == case["labels"]
    assert d1.tolist() == case["d1"]
    assert J == case["objective"]
    assert oracle.objective(X, C0, labels) == case["objective"]
    C1, counts, nr = oracle.update(X, labels, d1, C0)
    assert C1.tolist() == case["C1"]
    assert counts.tolist() == case["counts"]
    assert nr == sum(1 for c in case["counts"] if c == 0)


def test_duplicate_centres_lowest_index():
    X = np.random.RandomState(3).randn(300, 4).astype(np.float32)
    C = np.stack([np.zeros(4), np.zeros(4), np.full(4, 50.0), np.zeros(4)]).astype(np.float32)
    labels, d1, d2, _ = oracle.assign(X, C)
    assert set(labels.tolist()) == {0}
    assert np.array_equal(d1, d2)  # the duplicate is the runner-up at the same distance


# ----------------------------------------------------------------------------------
# brute force and exact optima
# ----------------------------------------------------------------------------------

def _brute_force_opt(X, K):
    n = X.shape[0]
    best, arg = math.inf, None
    Xd = X.astype(np.float64)
    for lab in itertools.product(range(K), repeat=n):
        lab = np.array(lab)
        J = 0.0
        for k in range(K):
            m = lab == k
            if m.any():
                J += float(((Xd[m] - Xd[m].mean(0)) ** 2).sum())
        if J < best - 1e-12:
            best, arg = J, lab
    return best, arg


@pytest.mark.parametrize("seed", range(6))
def test_brute_force_optimum(seed):
    rng = np.random.RandomState(100 + seed)
    n, K, d = 7, 3, 1 + seed % 3
    X = rng.randn(n, d).astype(np.float32) * 2
    Jstar, lab = _brute_force_opt(X, K)
    # 1) Lloyd never goes below the optimum, whatever the start
    C0, _ = oracle.kmeanspp(X, K, seed)
    C, labels, objs, _, _ = oracle.lloyd(X, C0, 8)
    _, _, _, Jend = oracle.assign(X, C)
    assert Jend >= Jstar * (1 - 1e-9) - 1e-12
    assert min(objs) >= Jstar * (1 - 1e-9) - 1e-12
    # 2) the optimum's centres are a fixed point of Lloyd's iteration
    Copt = np.stack([X[lab == k].astype(np.float64).mean(0) for k in range(K)]).astype(np.float32)
    C2, labels2, objs2, changed2, _ = oracle.lloyd(X, Copt, 3)
    assert np.allclose(objs2, Jstar, rtol=1e-6)
    assert np.array_equal(labels2, lab)
    assert np.array_equal(C2, Copt)


@pytest.mark.parametrize("seed", range(3))
def test_brute_force_separated_reaches_optimum(seed):
    rng = np.random.RandomState(200 + seed)
    centers = np.array([[0, 0], [30, 0], [0, 30]], np.float32)
    comp = np.concatenate([[0, 1, 2], rng.randint(0, 3, 5)])  # every group present
    X = (centers[comp] + rng.randn(8, 2)).astype(np.float32)
    Jstar, _ = _brute_force_opt(X, 3)
    C0, _ = oracle.kmeanspp(X, 3, seed)
    C, _, _, _, _ = oracle.lloyd(X, C0, 6)
    _, _, _, J = oracle.assign(X, C)
    assert J == pytest.approx(Jstar, rel=1e-9, abs=1e-9)


def _dp_1d(x, K):
    """Exact 1-D K-means optimum by dynamic programming over sorted points (Wang & Song 2011)."""
    x = np.sort(np.asarray(x, np.float64))
    n = len(x)
    s1 = np.concatenate([[0.0], np.cumsum(x)])
    s2 = np.concatenate([[0.0], np.cumsum(x * x)])

    def cost(a, b):  # points a..b inclusive
        m = b - a + 1
        t = s1[b + 1] - s1[a]
        return (s2[b + 1] - s2[a]) - t * t / m

    D = np.full((K + 1, n), np.inf)
    for i in range(n):
        D[1, i] = cost(0, i)
    for k in range(2, K + 1):
        for i in range(k - 1, n):
            D[k, i] = min(D[k - 1, j - 1] + cost(j, i) for j in range(k - 1, i + 1))
    return D[K, n - 1]


@pytest.mark.parametrize("K", [2, 3, 5])
def test_1d_exact_optimum(K):
    rng = np.random.RandomState(K)
    # well-separated groups: Lloyd from k-means++ (best of a few seeds) reaches the optimum
    centers = np.arange(K) * 40.0
    x = (centers[rng.randint(0, K, 200)] + rng.randn(200)).astype(np.float32)
    x[:K] = centers
    X = x[:, None]
    opt = _dp_1d(x, K)
    best = math.inf
    for s in range(4):
        C0, _ = oracle.kmeanspp(X, K, 1000 + s)
        C, _, objs, _, _ = oracle.lloyd(X, C0, 20)
        _, _, _, J = oracle.assign(X, C)
        assert J >= opt * (1 - 1e-9)
        best = min(best, J)
    assert best == pytest.approx(opt, rel=1e-7)
    # on unstructured data Lloyd can stop above the optimum but never below it
    xr = rng.rand(150).astype(np.float32)
    C0, _ = oracle.kmeanspp(xr[:, None], K, 7)
    C, _, _, _, _ = oracle.lloyd(xr[:, None], C0, 10)
    _, _, _, J = oracle.assign(xr[:, None], C)
    assert J >= _dp_1d(xr, K) * (1 - 1e-9)


# ----------------------------------------------------------------------------------
# closed forms and special cases
# ----------------------------------------------------------------------------------

def test_k1_global_mean_and_total_scatter():
    X = (np.random.RandomState(5).randn(500, 7) * 3 + 1).astype(np.float32)
    C0 = np.zeros((1, 7), np.float32)
    labels, d1, _, _ = oracle.assign(X, C0)
    C1, counts, _ = oracle.update(X, labels, d1, C0)
    Xd = X.astype(np.float64)
    mean = np.array([math.fsum(Xd[:, j]) / 500 for j in range(7)])
    assert np.array_equal(C1[0], mean.astype(np.float32))
    _, _, d2, J = oracle.assign(X, C1)
    assert np.all(np.isinf(d2))
    # J = sum ||x||^2 - N ||mean||^2, evaluated with the fp32 centre actually used
    c = C1[0].astype(np.float64)
    J_identity = math.fsum((Xd ** 2).ravel()) - 2 * float(Xd.sum(0) @ c) + 500 * float(c @ c)
    assert J == pytest.approx(J_identity, rel=1e-10)
    assert counts.tolist() == [500]


def test_k_equals_n_zero_objective():
    X = np.random.RandomState(6).randn(12, 3).astype(np.float32)
    C0, picked = oracle.kmeanspp(X, 12, 99)
    assert sorted(picked.tolist()) == list(range(12))  # D^2 sampling never repeats a chosen point
    assert np.array_equal(C0, X[picked])
    labels, d1, _, J = oracle.assign(X, C0)
    assert J == 0.0
    assert np.array_equal(picked[labels], np.arange(12))


def test_closed_form_well_separated_mixture():
    """Config 1 recipe: 16 centres ~ N(0, 16 I) in d = 128, unit noise.

    Started from the generating components' means, Lloyd keeps the generating
    partition, and E[J] = sum_k (n_k - 1) d = (N - K) d, so J / (N d) is
    1 - K/N up to chi-square noise of sd sqrt(2 / (N d)).
    """
    w = hme_synth.WORKLOADS[1]
    X, comp = hme_synth.make_features(w)
    X = X.numpy()
    comp = comp.numpy()
    C0 = np.stack([X[comp == k].astype(np.float64).mean(0) for k in range(w.K)]).astype(np.float32)
    C, labels, objs, changed, counts = oracle.lloyd(X, C0, 3)
    assert np.array_equal(labels, comp)
    assert counts.tolist() == np.bincount(comp, minlength=w.K).tolist()
    ratio = objs[-1] / (w.N * w.d)
    assert abs(ratio - (1 - w.K / w.N)) < 6 * math.sqrt(2 / (w.N * w.d))
    assert changed[1:].tolist() == [0, 0]


# ----------------------------------------------------------------------------------
# invariants of Lloyd's iteration
# ----------------------------------------------------------------------------------

def test_lloyd_invariants_random_data():
    rng = np.random.RandomState(8)
    X = (rng.randn(800, 6) + rng.randint(0, 3, (800, 1)) * 2.5).astype(np.float32)
    K = 9
    C, _ = oracle.kmeanspp(X, K, 3)
    Xd = X.astype(np.float64)
    prevJ = math.inf
    for t in range(6):
        labels, d1, d2, J = oracle.assign(X, C)
        # monotone non-increase of the objective
        assert J <= prevJ * (1 + 1e-12)
        prevJ = J
        # exact nearest centre, re-evaluated with the norm expansion in a different order
        Cd = C.astype(np.float64)
        D = (Xd ** 2).sum(1)[:, None] - 2 * Xd @ Cd.T + (Cd ** 2).sum(1)[None, :]
        Ds = np.sort(D, 1)
        scale = 1e-9 * (1 + D.max())
        assert np.all(D[np.arange(800), labels] <= Ds[:, 0] + scale)
        assert np.allclose(d1, Ds[:, 0], atol=scale)
        assert np.allclose(d2, Ds[:, 1], atol=scale)
        # lowest index among exact minima
        for i in np.where(np.abs(Ds[:, 1] - Ds[:, 0]) <= scale)[0]:
            assert labels[i] == np.where(np.abs(D[i] - Ds[i, 0]) <= scale)[0].min()
        # the objective of the assign's own labels is the assign's objective; any other labelling is not lower
        assert oracle.objective(X, C, labels) == J
        assert oracle.objective(X, C, (labels + 1) % K) >= J
        C_new, counts, nr = oracle.update(X, labels, d1, C)
        assert counts.sum() == 800
        assert counts.tolist() == np.bincount(labels, minlength=K).tolist()
        for k in range(K):
            if counts[k]:
                m = Xd[labels == k]
                exact = np.array([math.fsum(m[:, j]) for j in range(6)]) / counts[k]
                assert np.allclose(C_new[k], exact, rtol=2 ** -23, atol=1e-30)
        C = C_new


def test_lloyd_objective_sequence_monotone():
    w = hme_synth.WORKLOADS[2].with_rows(3000)
    X, _ = hme_synth.make_features(dataclass_small(w))
    X = X.numpy()
    C0, _ = oracle.kmeanspp(X, 8, 11, subsample=True)
    _, _, objs, changed, _ = oracle.lloyd(X, C0, 8)
    assert np.all(np.diff(objs) <= 1e-12 * objs[:-1])
    assert changed[0] == X.shape[0]


def dataclass_small(w):
    import dataclasses
    return dataclasses.replace(w, d=48, comps=8)


def test_reseed_order_and_no_reuse():
    # three empty clusters share tied distances: ascending k takes ascending i among equal mind
    X = np.array([[0, 0], [2, 0], [0, 2], [-2, 0], [0, -2]], np.float32)
    C0 = np.array([[0, 0], [90, 90], [91, 91], [92, 92]], np.float32)
    labels, d1, _, _ = oracle.assign(X, C0)
    C1, counts, nr = oracle.update(X, labels, d1, C0)
    assert nr == 3 and counts.tolist() == [5, 0, 0, 0]
    assert C1[1:].tolist() == [[2, 0], [0, 2], [-2, 0]]
    # more empty clusters than points: the rest keep their old centre
    X2 = np.array([[1, 1]], np.float32)
    C2, counts2, nr2 = oracle.update(X2, np.array([0], np.int32), np.array([2.0]), C0)
    assert nr2 == 1 and C2[1].tolist() == [1, 1] and C2[2].tolist() == [91, 91]


# ----------------------------------------------------------------------------------
# k-means++ (Arthur & Vassilvitskii 2007): D^2 sampling, checked statistically
# ----------------------------------------------------------------------------------

def test_kmeanspp_d2_sampling_distribution():
    from scipy.stats import chisquare
    x = np.array([0.0, 1.0, 3.0, 7.0, 15.0], np.float32)[:, None]
    n, S = 5, 20000
    obs = np.zeros((n, n))
    for s in range(S):
        _, picked = oracle.kmeanspp(x, 2, s)
        obs[picked[0], picked[1]] += 1
    exp = np.zeros((n, n))
    for f in range(n):
        d2 = (x[:, 0].astype(np.float64) - x[f, 0]) ** 2
        exp[f] = S / n * d2 / d2.sum()
    mask = exp > 0
    assert obs[~mask].sum() == 0  # never re-picks the first centre
    assert chisquare(obs[mask], exp[mask]).pvalue > 1e-4
    assert chisquare(obs.sum(1), np.full(n, S / n)).pvalue > 1e-4


def test_kmeanspp_first_pick_and_rows():
    X = np.random.RandomState(9).randn(1000, 5).astype(np.float32)
    for seed in [0, 1, 12345]:
        C, picked = oracle.kmeanspp(X, 6, seed)
        assert picked[0] == oracle.scaled_index(oracle.splitmix64_at(seed, 0), 1000)
        assert np.array_equal(C, X[picked])
        assert len(set(picked.tolist())) == 6
        # with N <= 256 K the subsample is every row, so both modes agree
        C2, picked2 = oracle.kmeanspp(X, 6, seed, subsample=True)
        assert np.array_equal(picked, picked2)
    # subsample mode on N > 256 K still returns real rows of X
    C3, picked3 = oracle.kmeanspp(X, 3, 5, subsample=True)
    assert np.array_equal(C3, X[picked3]) and picked3.max() < 1000


def test_bf16_assign_uses_rounded_centres():
    rng = np.random.RandomState(10)
    Xf = torch.from_numpy(rng.randn(400, 33).astype(np.float32)).to(torch.bfloat16)
    C = rng.randn(7, 33).astype(np.float32)
    lab_b, d1_b, d2_b, J_b = oracle.assign(hme_synth.bf16_bits(Xf), C, dtype="bf16")
    C_r = torch.from_numpy(C).to(torch.bfloat16).float().numpy()
    lab_f, d1_f, d2_f, J_f = oracle.assign(Xf.float().numpy(), C_r, dtype="f32")
    assert np.array_equal(lab_b, lab_f) and np.array_equal(d1_b, d1_f) and J_b == J_f


# ----------------------------------------------------------------------------------
# partition: stable counting sort == numpy's stable argsort (a library routine)
# ----------------------------------------------------------------------------------

@pytest.mark.parametrize("K", [1, 5, 37, 300])
def test_partition_matches_stable_argsort(K):
    rng = np.random.RandomState(K)
    w = np.arange(1, K + 1, dtype=np.float64) ** -1.1
    labels = rng.choice(K, size=5000, p=w / w.sum()).astype(np.int32)
    out = oracle.partition(labels, K)
    assert np.array_equal(out["perm"], np.argsort(labels, kind="stable"))
    assert np.array_equal(out["hist"], np.bincount(labels, minlength=K))
    assert np.array_equal(out["offsets"], np.concatenate([[0], np.cumsum(np.bincount(labels, minlength=K))]))
    assert np.array_equal(out["sorted_labels"], np.sort(labels))
    assert sorted(out["perm"].tolist()) == list(range(5000))


def test_partition_moves_tag_lists():
    rng = np.random.RandomState(12)
    N, K = 400, 6
    labels = rng.randint(0, K, N).astype(np.int32)
    lists = [rng.randint(0, 50, rng.poisson(3)).tolist() for _ in range(N)]
    tag_off = np.concatenate([[0], np.cumsum([len(l) for l in lists])]).astype(np.int64)
    tags = np.array([t for l in lists for t in l], np.int32)
    out = oracle.partition(labels, K, tag_off, tags)
    order = sorted(range(N), key=lambda i: (labels[i], i))
    exp_tags = [t for i in order for t in lists[i]]
    exp_off = np.concatenate([[0], np.cumsum([len(lists[i]) for i in order])])
    assert out["tags"].tolist() == exp_tags
    assert out["tag_off"].tolist() == exp_off.tolist()


def test_partition_rejects_bad_labels():
    with pytest.raises(ValueError):
        oracle.partition(np.array([0, 3, 1], np.int32), 3)
    with pytest.raises(ValueError):
        oracle.partition(np.array([0, -1], np.int32), 3)
    with pytest.raises(ValueError):
        oracle.update(np.zeros((2, 2), np.float32), np.array([0, 5], np.int32), None, np.zeros((2, 2), np.float32))


def test_empty_input():
    out = oracle.partition(np.zeros(0, np.int32), 4)
    assert out["hist"].tolist() == [0, 0, 0, 0] and out["offsets"].tolist() == [0] * 5


# ---------------------------------------------------------------------------
# Tag statistics of a clustering (Section 4.5)
# ---------------------------------------------------------------------------
TAG_CASES = json.load(open(os.path.join(GOLDEN, "tag_cluster_hand_examples.json")))["cases"]


@pytest.mark.parametrize("case", TAG_CASES, ids=lambda c: c["name"])
def test_tag_hist_hand_examples(case):
    counts, sp = oracle.tag_cluster_hist(np.array(case["labels"], np.int32), case["K"],
                                         np.array(case["tag_off"], np.int64), np.array(case["tags"], np.int32),
                                         case["V"])
    assert np.array_equal(counts, np.array(case["counts"], np.int64))
    assert np.allclose(sp, case["sparsity"], rtol=1e-15, atol=0)


def _random_tagged(N, K, V, seed):
    rng = np.random.default_rng(seed)
    labels = rng.integers(0, K, N).astype(np.int32)
    lens = rng.poisson(3.0, N)
    tag_off = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    # Zipf-like vocabulary: a few tags very common
    w = 1.0 / np.arange(1, V + 1)
    tags = rng.choice(V, int(tag_off[-1]), p=w / w.sum()).astype(np.int32)
    return labels, tag_off, tags


def test_tag_hist_marginals():
    """Row sums = tags carried by each cluster's points; column sums = occurrences of each tag."""
    N, K, V = 3000, 17, 200
    labels, tag_off, tags = _random_tagged(N, K, V, 3)
    counts, sp = oracle.tag_cluster_hist(labels, K, tag_off, tags, V)
    lens = np.diff(tag_off)
    per_cluster = np.array([lens[labels == k].sum() for k in range(K)])
    assert np.array_equal(counts.sum(1), per_cluster)
    assert np.array_equal(counts.sum(0), np.bincount(tags, minlength=V))
    present = counts.sum(0) > 0
    assert np.all(sp[~present] == 0.0)
    # ||c||_1 / ||c||_2 lies in [1, sqrt(number of clusters the tag occurs in)]
    nz = (counts > 0).sum(0)
    assert np.all(sp[present] >= 1.0 - 1e-12)
    assert np.all(sp[present] <= np.sqrt(nz[present]) + 1e-12)


def test_tag_hist_closed_forms():
    """A tag confined to one cluster has sparsity 1; equal counts over m clusters give sqrt(m)."""
    K, V = 9, 4
    labels, offs, tags = [], [0], []
    for k in range(K):
        for _ in range(5):  # five points per cluster
            labels.append(k)
            t = [0] if k < 6 else []          # tag 0: once per point in clusters 0..5 -> m = 6
            t += [1, 1] if k == 4 else []     # tag 1: only in cluster 4
            t += [3] * (k + 1)                # tag 3: counts 5 (k + 1) per cluster, unequal
            tags += t
            offs.append(offs[-1] + len(t))
    counts, sp = oracle.tag_cluster_hist(np.array(labels, np.int32), K, np.array(offs, np.int64),
                                         np.array(tags, np.int32), V)
    assert sp[0] == pytest.approx(np.sqrt(6.0), rel=1e-15)
    assert sp[1] == 1.0
    assert sp[2] == 0.0
    c3 = 5.0 * np.arange(1, K + 1)
    assert sp[3] == pytest.approx(c3.sum() / np.sqrt((c3 ** 2).sum()), rel=1e-15)


def test_tag_hist_invariant_under_point_order():
    """The statistics depend on (label, tags) pairs only: the partitioned order gives the same result."""
    N, K, V = 2000, 11, 150
    labels, tag_off, tags = _random_tagged(N, K, V, 8)
    counts, sp = oracle.tag_cluster_hist(labels, K, tag_off, tags, V)
    part = oracle.partition(labels, K, tag_off, tags)
    counts2, sp2 = oracle.tag_cluster_hist(part["sorted_labels"], K, part["tag_off"], part["tags"], V)
    assert np.array_equal(counts, counts2)
    assert np.array_equal(sp, sp2)


def test_tag_hist_rejects_out_of_range():
    with pytest.raises(ValueError):
        oracle.tag_cluster_hist(np.array([0, 3], np.int32), 3, np.array([0, 1, 2]), np.array([0, 1], np.int32), 2)
    with pytest.raises(ValueError):
        oracle.tag_cluster_hist(np.array([0, 1], np.int32), 3, np.array([0, 1, 2]), np.array([0, 2], np.int32), 2)
