"""Seeded synthetic feature sets shaped like the gater's input.

The paper clusters pooled last-hidden-layer CNN features of YFCC100M (about
100M images) and of a private 440M-image Instagram set, projected to 256 PCA
dimensions with K = 50 (Section 4, "YFCC100M", "Instagram Food", Section 4.2).
Those datasets and trained trunks are not available, so these generators stand
in for them: Gaussian mixtures (optionally post-ReLU, L2-normalised or
Zipf-skewed in component weight) with the sizes of the five workloads below.

This module holds NO arithmetic of the method (no distances, no argmin, no
means, no partition).  It is shared by the tests (which feed the same bytes to
the oracle and to the CUDA path) and by bench.py.  Random numbers come from
torch generators seeded per workload; data may be generated on the GPU and
copied to the host for the oracle.
"""
from __future__ import annotations

import dataclasses
from typing import Optional

import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    N: int
    d: int
    K: int
    dtype: str            # "f32" or "bf16": element type of the feature matrix
    comps: int            # mixture components
    center_std: float
    noise_std: float
    zipf: float           # 0 = uniform component weights, else weight_k ~ (k+1)^-zipf
    relu: bool            # pooled post-ReLU features: x = max(0, z)
    l2norm: bool          # rows scaled to unit L2 norm
    iters: int            # Lloyd iterations
    seed: int
    init_subsample: bool  # k-means++ on a subsample of min(N, 256 K) rows
    tags: bool = False    # carries a CSR multilabel list per point
    tag_mean: float = 3.0
    tag_vocab: int = 20000
    tag_zipf: float = 1.0
    route: bool = False   # the job ends with a route (assign + partition) pass

    def with_rows(self, N: int) -> "Workload":
        """The same recipe with fewer points (a seeded row-subsample stand-in)."""
        return dataclasses.replace(self, N=int(N))

    @property
    def elem_bytes(self) -> int:
        return 4 if self.dtype == "f32" else 2


WORKLOADS = {
    # 16 well-separated Gaussians, centres ~ N(0, 4^2 I), unit noise, seed 0.
    1: Workload("gmm16_n1e4_d128_k16_f32", 10_000, 128, 16, "f32", 16, 4.0, 1.0, 0.0, False, False, 10, 0, False),
    # ResNet-50-like pooled features: max(0, z), z ~ mixture of 64 Gaussians, about half zeros.
    2: Workload("relu_gmm64_n1e6_d2048_k64_f32", 1_000_000, 2048, 64, "f32", 64, 1.0, 1.0, 0.0, True, False, 20, 1,
                True, route=True),
    # Post-ReLU mixture of 256 with Zipf(1.1) weights (largest component about 21%).
    3: Workload("relu_zipf256_n4e6_d2048_k256_bf16", 4_000_000, 2048, 256, "bf16", 256, 1.0, 1.0, 1.1, True, False,
                20, 2, True),
    # Random-projected, L2-normalised features with Poisson(3) tags from a Zipf(1.0) vocabulary of 20000.
    4: Workload("l2_gmm1024_n16e6_d512_k1024_f32", 16_000_000, 512, 1024, "f32", 1024, 1.0, 1.0, 0.0, False, True,
                10, 3, True, tags=True),
    # 4096 Gaussians with Zipf(1.0) weights, 26 GB of bf16 features resident in HBM.
    5: Workload("zipf4096_n5e7_d256_k4096_bf16", 50_000_000, 256, 4096, "bf16", 4096, 1.0, 1.0, 1.0, False, False,
                5, 4, True),
}

_CHUNK_ROWS = 1 << 20


def _gen(device, seed: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed) & ((1 << 63) - 1))
    return g


def _categorical(weights: torch.Tensor, n: int, g: torch.Generator, device) -> torch.Tensor:
    """n draws from a categorical distribution by inverse CDF (searchsorted)."""
    cdf = torch.cumsum(weights.double(), 0)
    cdf = (cdf / cdf[-1]).to(device)
    u = torch.rand(n, generator=g, device=device, dtype=torch.float64)
    return torch.searchsorted(cdf, u, right=True).clamp_(max=weights.numel() - 1)


def component_weights(w: Workload) -> torch.Tensor:
    if w.zipf == 0.0:
        return torch.ones(w.comps, dtype=torch.float64)
    return torch.arange(1, w.comps + 1, dtype=torch.float64).pow(-w.zipf)


def make_features(w: Workload, device="cpu", N: Optional[int] = None, out: Optional[torch.Tensor] = None):
    """Feature matrix (N, d): float32, or bfloat16 for bf16 workloads.

    Returns (X, comp) where comp[i] is the generating component of row i (kept
    for closed-form checks; the method never sees it).
    """
    N = w.N if N is None else int(N)
    device = torch.device(device)
    tdt = torch.float32 if w.dtype == "f32" else torch.bfloat16
    g = _gen(device, 0x5EED0000 + w.seed)
    centers = torch.randn(w.comps, w.d, generator=g, device=device, dtype=torch.float32) * w.center_std
    weights = component_weights(w)
    X = out if out is not None else torch.empty(N, w.d, dtype=tdt, device=device)
    comp = torch.empty(N, dtype=torch.int32, device=device)
    for c0 in range(0, N, _CHUNK_ROWS):
        n = min(_CHUNK_ROWS, N - c0)
        gc = _gen(device, (w.seed + 1) * 1_000_003 + c0 // _CHUNK_ROWS)
        cid = _categorical(weights, n, gc, device)
        z = centers[cid] + torch.randn(n, w.d, generator=gc, device=device, dtype=torch.float32) * w.noise_std
        if w.relu:
            z.clamp_(min=0.0)
        if w.l2norm:
            z = z / z.norm(dim=1, keepdim=True).clamp_(min=1e-12)
        X[c0:c0 + n].copy_(z.to(tdt))
        comp[c0:c0 + n] = cid.to(torch.int32)
    return X, comp


def make_tags(w: Workload, N: Optional[int] = None, device="cpu"):
    """CSR multilabel lists: tag_off int64[N+1], tags int32[T].

    Per point Poisson(tag_mean) tags; tag ids Zipf(tag_zipf) over tag_vocab words.
    """
    N = w.N if N is None else int(N)
    device = torch.device(device)
    g = _gen(device, 0x7A60000 + w.seed)
    rates = torch.full((N,), float(w.tag_mean), device=device, dtype=torch.float32)
    counts = torch.poisson(rates, generator=g).to(torch.int64)
    tag_off = torch.zeros(N + 1, dtype=torch.int64, device=device)
    torch.cumsum(counts, 0, out=tag_off[1:])
    T = int(tag_off[-1].item())
    vocab_w = torch.arange(1, w.tag_vocab + 1, dtype=torch.float64).pow(-w.tag_zipf)
    tags = torch.empty(T, dtype=torch.int32, device=device)
    for t0 in range(0, T, 1 << 24):
        n = min(1 << 24, T - t0)
        tags[t0:t0 + n] = _categorical(vocab_w, n, g, device).to(torch.int32)
    return tag_off, tags


def bf16_bits(X: torch.Tensor):
    """Host numpy uint16 view of a bfloat16 tensor (how the oracle takes bf16)."""
    return X.detach().to("cpu").contiguous().view(torch.int16).numpy().view("uint16")


def host_array(X: torch.Tensor, dtype: str):
    """Host numpy array of a feature tensor in the oracle's convention."""
    if dtype == "bf16":
        return bf16_bits(X)
    return X.detach().to("cpu").contiguous().numpy()


def random_centroids(K: int, d: int, seed: int, scale: float = 1.0, device="cpu"):
    """Arbitrary fp32 centres for teacher-forced single-step checks."""
    g = _gen(torch.device(device), 0xC0FFEE + seed)
    return torch.randn(K, d, generator=g, device=device, dtype=torch.float32) * scale


def expected_zero_fraction(w: Workload) -> float:
    """For post-ReLU sets with centre and noise std s_c, s_n: P(z <= 0) = 1/2."""
    return 0.5 if w.relu else 0.0


def component_sizes(w: Workload) -> torch.Tensor:
    """Expected points per component, N * weight (for skew checks)."""
    p = component_weights(w)
    return p / p.sum() * w.N


__all__ = ["Workload", "WORKLOADS", "make_features", "make_tags", "bf16_bits", "host_array", "random_centroids",
           "component_sizes", "expected_zero_fraction"]
