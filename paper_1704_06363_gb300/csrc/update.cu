// update.cu -- the K-means centre step (Section 2: the gater's centres come
// from "K-means clustering" of the z_j) and the empty-cluster rule.
//
//   sums      rows are visited in the stable sorted order of their labels
//             (perm / sorted_labels from the partition kernels), so each
//             cluster is a contiguous segment.  A CTA owns a contiguous range
//             of that order and, per thread, one 16-byte column vector of the
//             rows; it adds rows into fp32 registers and flushes to the fp64
//             global sums with one atomic per element each time the segment
//             (label) changes and at the end of its range.  Reads are whole
//             16-byte vectors of contiguous rows (coalesced across the CTA);
//             four rows are in flight per thread.  The same pass adds
//             (x - c_t[label])^2 by direct differences: the Lloyd objective of
//             (C_t, labels), free of the cancellation of the norm expansion.
//   finalize  c_k = sums_k / counts_k (fp64 divide, rounded once to fp32) for
//             non-empty k; counts_out = counts.
//   reseed    one CTA: in ascending k, every empty cluster takes the row that
//             comes next in the order (mind descending, index ascending), i.e.
//             the farthest point not yet taken, ties to the lowest index.  The
//             row is copied exactly into c_k.  Nothing runs when no cluster is
//             empty beyond one scan of the counts.
#include "hme_common.cuh"

namespace hme {

namespace {

template <int DT, int VW>
struct Vec;
template <>
struct Vec<HME_F32, 4> {
  static __device__ __forceinline__ void load(const void *base, int64_t off, float (&v)[4]) {
    float4 f;
    asm volatile("ld.global.nc.L1::no_allocate.v4.f32 {%0,%1,%2,%3}, [%4];"
                 : "=f"(f.x), "=f"(f.y), "=f"(f.z), "=f"(f.w)
                 : "l"(static_cast<const float *>(base) + off));
    v[0] = f.x, v[1] = f.y, v[2] = f.z, v[3] = f.w;
  }
};
template <>
struct Vec<HME_F32, 1> {
  static __device__ __forceinline__ void load(const void *base, int64_t off, float (&v)[1]) {
    v[0] = __ldg(static_cast<const float *>(base) + off);
  }
};
template <>
struct Vec<HME_BF16, 8> {
  static __device__ __forceinline__ void load(const void *base, int64_t off, float (&v)[8]) {
    uint4 u;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(u.x), "=r"(u.y), "=r"(u.z), "=r"(u.w)
                 : "l"(static_cast<const __nv_bfloat16 *>(base) + off));
    const __nv_bfloat162 *h = reinterpret_cast<const __nv_bfloat162 *>(&u);
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const float2 f = __bfloat1622float2(h[t]);
      v[2 * t] = f.x, v[2 * t + 1] = f.y;
    }
  }
};
template <>
struct Vec<HME_BF16, 1> {
  static __device__ __forceinline__ void load(const void *base, int64_t off, float (&v)[1]) {
    v[0] = __bfloat162float(static_cast<const __nv_bfloat16 *>(base)[off]);
  }
};

constexpr int kUpdThreads = 256;
constexpr int kUnroll = 4;

// Block layout: G groups of V threads; thread (g, t) owns column vector
// (blockIdx.y * V + t) and the g-th sub-range of the block's row range.
// Besides the sums, every thread adds (x - c_t[label])^2 over its elements,
// c_t being the centres before this update (bf16-rounded for bf16 features,
// the values the assign step compared against): the Lloyd objective of
// (C_t, labels) by direct differences.  fp32 partials are folded into fp64
// every 64 rows and at the end, then reduced once per block.
template <int DT, int VW>
__global__ void __launch_bounds__(kUpdThreads) update_sums_kernel(const void *__restrict__ X, int64_t N, int d,
                                                                  int64_t ldx, const int32_t *__restrict__ perm,
                                                                  const int32_t *__restrict__ slab,
                                                                  const int64_t *__restrict__ valid_total, int V,
                                                                  int G, int64_t rows_per_block, double *sums,
                                                                  const float *__restrict__ Cold, double *Jsum) {
  __shared__ double jpart[kUpdThreads / 32];
  const int g = threadIdx.x / V;
  const int t = threadIdx.x - g * V;
  const int vcol = blockIdx.y * V + t;
  const int col = vcol * VW;
  const int64_t b0 = (int64_t)blockIdx.x * rows_per_block;
  const int64_t b1 = min(min(N, *valid_total), b0 + rows_per_block);
  const int64_t per = (b1 - b0 + G - 1) / G;
  const int64_t r0 = b0 + g * per;
  const int64_t r1 = min(b1, r0 + per);
  const bool active = (g < G) && (col < d) && (r0 < r1);
  double jd = 0.0;

  if (active) {
    float acc[VW], cc[VW];
    float accj = 0.0f;
    int cur = __ldg(slab + r0);
    auto load_centre = [&](int lab) {
#pragma unroll
      for (int e = 0; e < VW; ++e) {
        const float c = (VW == 1 || col + e < d) ? __ldg(Cold + (int64_t)lab * d + col + e) : 0.0f;
        cc[e] = (DT == HME_BF16) ? __bfloat162float(__float2bfloat16_rn(c)) : c;
      }
    };
    auto flush = [&](int lab) {
      double *dst = sums + (int64_t)lab * d + col;
#pragma unroll
      for (int e = 0; e < VW; ++e) {
        if (VW == 1 || col + e < d) atomicAdd(dst + e, (double)acc[e]);
        acc[e] = 0.0f;
      }
    };
    auto add_row = [&](const float (&v)[VW]) {
#pragma unroll
      for (int e = 0; e < VW; ++e) {
        acc[e] += v[e];
        const float q = v[e] - cc[e];
        accj = fmaf(q, q, accj);
      }
    };
#pragma unroll
    for (int e = 0; e < VW; ++e) acc[e] = 0.0f;
    load_centre(cur);

    int64_t j = r0;
    int since = 0;
    for (; j + kUnroll <= r1; j += kUnroll) {
      int lab[kUnroll];
      float v[kUnroll][VW];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int64_t row = __ldg(perm + j + u);
        lab[u] = __ldg(slab + j + u);
        Vec<DT, VW>::load(X, row * ldx + col, v[u]);
      }
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        if (lab[u] != cur) {
          flush(cur);
          cur = lab[u];
          load_centre(cur);
        }
        add_row(v[u]);
      }
      if ((since += kUnroll) >= 64) {
        jd += (double)accj;
        accj = 0.0f;
        since = 0;
      }
    }
    for (; j < r1; ++j) {
      const int64_t row = __ldg(perm + j);
      const int lab = __ldg(slab + j);
      float v[VW];
      Vec<DT, VW>::load(X, row * ldx + col, v);
      if (lab != cur) {
        flush(cur);
        cur = lab;
        load_centre(cur);
      }
      add_row(v);
    }
    flush(cur);
    jd += (double)accj;
  }

  // one fp64 atomic per block for the objective
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) jd += __shfl_xor_sync(0xffffffffu, jd, o);
  if ((threadIdx.x & 31) == 0) jpart[threadIdx.x >> 5] = jd;
  __syncthreads();
  if (threadIdx.x == 0) {
    double s = 0.0;
    for (int w = 0; w < kUpdThreads / 32; ++w) s += jpart[w];
    if (s != 0.0) atomicAdd(Jsum, s);
  }
}

__global__ void update_finalize_kernel(const double *__restrict__ sums, const int64_t *__restrict__ hist, int K,
                                       int d, float *__restrict__ C, int64_t *__restrict__ counts_out) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < (int64_t)K * d) {
    const int k = (int)(i / d);
    const int64_t n = hist[k];
    if (n > 0) C[i] = (float)(sums[i] / (double)n);
  }
  if (counts_out && i < K) counts_out[i] = hist[i];
}

// Order used by the re-seed rule: a comes before b if a is farther, or equally far with a lower index.
__device__ __forceinline__ bool before(float va, int64_t ia, float vb, int64_t ib) {
  return va > vb || (va == vb && ia < ib);
}

template <int DT>
__global__ void __launch_bounds__(1024) update_reseed_kernel(const void *__restrict__ X, int64_t N, int d,
                                                             int64_t ldx, const float *__restrict__ mind,
                                                             const int64_t *__restrict__ hist, int K, float *C,
                                                             int32_t *n_reseeded) {
  __shared__ float sv[32];
  __shared__ int64_t si[32];
  __shared__ int64_t pick_i;
  __shared__ float pick_v;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  // Nothing to do unless some cluster is empty (checked in parallel).
  int any_empty = 0;
  for (int k = threadIdx.x; k < K; k += blockDim.x) any_empty |= (hist[k] == 0);
  if (!__syncthreads_or(any_empty)) {
    if (threadIdx.x == 0 && n_reseeded) *n_reseeded = 0;
    return;
  }
  float last_v = INFINITY;  // the previous pick; the next one comes strictly after it
  int64_t last_i = -1;
  int taken = 0;
  for (int k = 0; k < K; ++k) {
    if (hist[k] != 0) continue;
    if (taken >= N) break;
    float bv = -INFINITY;
    int64_t bi = -1;
    for (int64_t i = threadIdx.x; i < N; i += blockDim.x) {
      const float v = mind ? mind[i] : 0.0f;
      if (before(last_v, last_i, v, i) && (bi < 0 || before(v, i, bv, bi))) {
        bv = v;
        bi = i;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
      const int64_t oi = __shfl_xor_sync(0xffffffffu, bi, o);
      if (oi >= 0 && (bi < 0 || before(ov, oi, bv, bi))) {
        bv = ov;
        bi = oi;
      }
    }
    if (lane == 0) {
      sv[warp] = bv;
      si[warp] = bi;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      float v = sv[0];
      int64_t ii = si[0];
      for (int w = 1; w < (int)(blockDim.x >> 5); ++w)
        if (si[w] >= 0 && (ii < 0 || before(sv[w], si[w], v, ii))) {
          v = sv[w];
          ii = si[w];
        }
      pick_v = v;
      pick_i = ii;
    }
    __syncthreads();
    const int64_t r = pick_i;
    if (r < 0) break;
    for (int j = threadIdx.x; j < d; j += blockDim.x) {
      float x;
      if (DT == HME_BF16)
        x = __bfloat162float(static_cast<const __nv_bfloat16 *>(X)[r * ldx + j]);
      else
        x = static_cast<const float *>(X)[r * ldx + j];
      C[(int64_t)k * d + j] = x;
    }
    last_v = pick_v;
    last_i = r;
    ++taken;
    __syncthreads();
  }
  if (threadIdx.x == 0 && n_reseeded) *n_reseeded = taken;
}

template <int DT, int VW>
void launch_sums(const void *X, int64_t N, int d, int64_t ldx, const int32_t *perm, const int32_t *slab,
                 const int64_t *valid_total, double *sums, const float *Cold, double *Jsum, cudaStream_t s) {
  const int nvec = (d + VW - 1) / VW;
  int V, G, ny;
  if (nvec <= kUpdThreads) {
    V = (nvec + 31) / 32 * 32;
    G = kUpdThreads / V;
    ny = 1;
  } else {
    V = kUpdThreads;
    G = 1;
    ny = (nvec + kUpdThreads - 1) / kUpdThreads;
  }
  int64_t nx = ((int64_t)num_sms() * 8 + ny - 1) / ny;
  const int64_t min_rows = 64 * (int64_t)G;
  if (nx * min_rows > N) nx = (N + min_rows - 1) / min_rows;
  if (nx < 1) nx = 1;
  const int64_t rpb = (N + nx - 1) / nx;
  dim3 grid((unsigned)nx, (unsigned)ny);
  update_sums_kernel<DT, VW><<<grid, kUpdThreads, 0, s>>>(X, N, d, ldx, perm, slab, valid_total, V, G, rpb,
                                                                  sums, Cold, Jsum);
  count_launch();
}

}  // namespace

cudaError_t launch_update(const void *X, int64_t N, int d, int64_t ldx, int dtype, const int32_t *perm,
                          const int32_t *sorted_labels, const int64_t *hist, const int64_t *valid_total,
                          const float *mind, int K, double *sums, float *C, int64_t *counts_out, int32_t *n_reseeded,
                          Header *hdr, cudaStream_t s) {
  cudaError_t e = cudaMemsetAsync(sums, 0, (size_t)K * d * sizeof(double), s);
  if (e != cudaSuccess) return e;
  if (N > 0) {
    const bool al = (reinterpret_cast<uintptr_t>(X) & 15u) == 0;
    if (dtype == HME_F32) {
      if (al && d % 4 == 0 && ldx % 4 == 0)
        launch_sums<HME_F32, 4>(X, N, d, ldx, perm, sorted_labels, valid_total, sums, C, &hdr->objective, s);
      else
        launch_sums<HME_F32, 1>(X, N, d, ldx, perm, sorted_labels, valid_total, sums, C, &hdr->objective, s);
    } else {
      if (al && d % 8 == 0 && ldx % 8 == 0)
        launch_sums<HME_BF16, 8>(X, N, d, ldx, perm, sorted_labels, valid_total, sums, C, &hdr->objective, s);
      else
        launch_sums<HME_BF16, 1>(X, N, d, ldx, perm, sorted_labels, valid_total, sums, C, &hdr->objective, s);
    }
  }
  const int64_t tot = (int64_t)K * d > K ? (int64_t)K * d : K;
  update_finalize_kernel<<<(unsigned)((tot + 255) / 256), 256, 0, s>>>(sums, hist, K, d, C, counts_out);
  if (dtype == HME_F32)
    update_reseed_kernel<HME_F32><<<1, 1024, 0, s>>>(X, N, d, ldx, mind, hist, K, C, n_reseeded);
  else
    update_reseed_kernel<HME_BF16><<<1, 1024, 0, s>>>(X, N, d, ldx, mind, hist, K, C, n_reseeded);
  count_launch(2);
  return cudaGetLastError();
}

}  // namespace hme
