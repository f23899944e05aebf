// update.cu -- the K-means centre step (Section 2: the gater's centres come
// from "K-means clustering" of the z_j) and the empty-cluster rule.
//
// Per-cluster state lives in the workspace between calls: fp64 sums S_k,
// int64 counts n_k and sum_i ||x_i||^2.  Two ways to bring it to the labels
// of this iteration:
//   full        rows are visited in the stable sorted order of their labels
//               (perm / sorted_labels from the partition kernels), so each
//               cluster is a contiguous segment.  A CTA owns a contiguous range
//               of that order and, per thread, one 16-byte column vector of the
//               rows; it adds rows into fp32 registers, folds them into fp64
//               registers every 64 rows and flushes to the fp64 sums with one
//               atomic per element each time the segment (label) changes.
//               Reads are whole 16-byte vectors of contiguous rows.
//   incremental given the labels of the previous call on the same workspace,
//               only rows whose label changed are read: x is added to the new
//               cluster's sum and subtracted from the old one (fp64), counts
//               move by one.  Lloyd's centres are the same sums, so the result
//               equals the full pass up to fp64 rounding order; after the first
//               iterations well under 1% of the rows change.
// Then:
//   objective   J = sum ||x||^2 - 2 sum_k c_k . S_k + sum_k n_k ||c_k||^2 in
//               fp64 with the centres that entered this update (bf16-rounded
//               for bf16 features): the Lloyd objective of (C_t, labels).
//   finalize    c_k = S_k / n_k (fp64 divide, rounded once to fp32) for
//               non-empty k; counts_out = n.
//   reseed      one CTA: in ascending k, every empty cluster takes the row that
//               comes next in the order (mind descending, index ascending), i.e.
//               the farthest point not yet taken, ties to the lowest index.  The
//               row is copied exactly into c_k.  Nothing runs when no cluster is
//               empty beyond one parallel scan of the counts.
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
// (blockIdx.y * V + t) and the g-th sub-range of the block's row range.  The
// thread also sums x^2 over its elements (sum ||x||^2 of the valid rows).
template <int DT, int VW>
__global__ void __launch_bounds__(kUpdThreads) update_sums_kernel(const void *__restrict__ X, int64_t N, int d,
                                                                  int64_t ldx, const int32_t *__restrict__ perm,
                                                                  const int32_t *__restrict__ slab,
                                                                  const int64_t *__restrict__ valid_total, int V,
                                                                  int G, int64_t rows_per_block, double *sums,
                                                                  double *x2sum, float sign) {
  __shared__ double qpart[kUpdThreads / 32];
  const int g = threadIdx.x / V;
  const int t = threadIdx.x - g * V;
  const int vcol = blockIdx.y * V + t;
  const int col = vcol * VW;
  const int64_t nrows = min(N, *valid_total);
  // rows_per_block == 0: split the (device-side) row count evenly over the blocks
  const int64_t rpb = rows_per_block > 0 ? rows_per_block : (nrows + gridDim.x - 1) / gridDim.x;
  const int64_t b0 = (int64_t)blockIdx.x * rpb;
  const int64_t b1 = min(nrows, b0 + rpb);
  const int64_t per = (b1 - b0 + G - 1) / G;
  const int64_t r0 = b0 + g * per;
  const int64_t r1 = min(b1, r0 + per);
  const bool active = (g < G) && (col < d) && (r0 < r1);
  double qd = 0.0;

  if (active) {
    float acc[VW];
    double accd[VW];
    float q = 0.0f;
    int cur = __ldg(slab + r0);
    auto fold = [&]() {
#pragma unroll
      for (int e = 0; e < VW; ++e) {
        accd[e] += (double)acc[e];
        acc[e] = 0.0f;
      }
      qd += (double)q;
      q = 0.0f;
    };
    auto flush = [&](int lab) {
      fold();
      double *dst = sums + (int64_t)lab * d + col;
#pragma unroll
      for (int e = 0; e < VW; ++e) {
        if (VW == 1 || col + e < d) atomicAdd(dst + e, accd[e]);
        accd[e] = 0.0;
      }
    };
    auto add_row = [&](const float (&v)[VW]) {
#pragma unroll
      for (int e = 0; e < VW; ++e) {
        acc[e] += sign * v[e];
        q = fmaf(sign * v[e], v[e], q);
      }
    };
#pragma unroll
    for (int e = 0; e < VW; ++e) {
      acc[e] = 0.0f;
      accd[e] = 0.0;
    }

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
        }
        add_row(v[u]);
      }
      if ((since += kUnroll) >= 64) {
        fold();
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
      }
      add_row(v);
    }
    flush(cur);
  }

  // one fp64 atomic per block for sum ||x||^2
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) qd += __shfl_xor_sync(0xffffffffu, qd, o);
  if ((threadIdx.x & 31) == 0) qpart[threadIdx.x >> 5] = qd;
  __syncthreads();
  if (threadIdx.x == 0) {
    double sq = 0.0;
    for (int w = 0; w < kUpdThreads / 32; ++w) sq += qpart[w];
    if (sq != 0.0) atomicAdd(x2sum, sq);
  }
}

// Incremental update, in four small kernels over the label vectors:
//   delta_count  rows whose label changed, counted per new label (to add) and
//                per old label (to subtract); labels outside [0, K) count as
//                unassigned on either side;
//   delta_scan   exclusive prefix of both counts -> fill cursors and totals;
//   delta_fill   the changed rows grouped by label (order inside a group is
//                irrelevant for sums), as (row, label) lists;
// then the sums kernel runs over each list (sign +1 / -1), and delta_counts
// moves n_k by the difference of the two counts.
// Warp-aggregated increment: lanes with the same key add once, by the lowest
// lane, and each lane gets its own slot (base + rank among equal keys).
__device__ __forceinline__ int32_t warp_add(int32_t *ctr, int key, bool active) {
  const unsigned act = __ballot_sync(0xffffffffu, active);
  const unsigned peers = __match_any_sync(0xffffffffu, active ? key : -1) & act;
  const int lane = threadIdx.x & 31;
  int32_t base = 0;
  if (active && lane == __ffs(peers) - 1) base = atomicAdd(ctr + key, __popc(peers));
  base = __shfl_sync(0xffffffffu, base, active ? __ffs(peers) - 1 : lane);
  return base + __popc(peers & ((1u << lane) - 1u));
}

__global__ void __launch_bounds__(256) delta_count_kernel(const int32_t *__restrict__ labels,
                                                          const int32_t *__restrict__ prev, int64_t N, int K,
                                                          int32_t *hist_add, int32_t *hist_sub, Header *hdr) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  bool bad = false;
  // whole warps iterate together (the loop bound is rounded up to a warp)
  const int64_t Nw = (N + 31) / 32 * 32;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < Nw; i += stride) {
    int a = -1, b = -1;
    if (i < N) {
      a = __ldg(labels + i);
      b = __ldg(prev + i);
      if (a < 0 || a >= K) {
        bad = true;
        a = -1;
      }
      if (b < 0 || b >= K) b = -1;
    }
    const bool moved = a != b;
    warp_add(hist_add, a, moved && a >= 0);
    warp_add(hist_sub, b, moved && b >= 0);
  }
  if (bad) atomicOr(&hdr->status, (uint32_t)kStatusBadLabel);
}

__global__ void __launch_bounds__(1024) delta_scan_kernel(const int32_t *__restrict__ hist_add,
                                                          const int32_t *__restrict__ hist_sub, int K,
                                                          int32_t *cur_add, int32_t *cur_sub, int64_t *totals) {
  __shared__ int64_t wsum[32];
  for (int which = 0; which < 2; ++which) {
    const int32_t *h = which == 0 ? hist_add : hist_sub;
    int32_t *cur = which == 0 ? cur_add : cur_sub;
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int per = (K + 1023) / 1024;
    const int k0 = t * per, k1 = min(K, k0 + per);
    int64_t local = 0;
    for (int k = k0; k < k1; ++k) local += h[k];
    int64_t incl = local;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int64_t v = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += v;
    }
    if (lane == 31) wsum[warp] = incl;
    __syncthreads();
    if (warp == 0) {
      const int64_t w = wsum[lane];
      int64_t wi = w;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int64_t v = __shfl_up_sync(0xffffffffu, wi, o);
        if (lane >= o) wi += v;
      }
      wsum[lane] = wi - w;
    }
    __syncthreads();
    int64_t run = wsum[warp] + incl - local;
    for (int k = k0; k < k1; ++k) {
      cur[k] = (int32_t)run;
      run += h[k];
    }
    if (t == 1023) totals[which] = run;
    __syncthreads();
  }
}

__global__ void delta_report_kernel(const int64_t *totals, Header *hdr) {
  hdr->moved_rows = (uint32_t)min(totals[0], (int64_t)0xFFFFFFFF);
}

__global__ void __launch_bounds__(256) delta_fill_kernel(const int32_t *__restrict__ labels,
                                                         const int32_t *__restrict__ prev, int64_t N, int K,
                                                         int32_t *cur_add, int32_t *cur_sub, int32_t *add_rows,
                                                         int32_t *add_lab, int32_t *sub_rows, int32_t *sub_lab) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t Nw = (N + 31) / 32 * 32;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < Nw; i += stride) {
    int a = -1, b = -1;
    if (i < N) {
      a = __ldg(labels + i);
      b = __ldg(prev + i);
      if (a < 0 || a >= K) a = -1;
      if (b < 0 || b >= K) b = -1;
    }
    const bool moved = a != b;
    const bool add = moved && a >= 0, sub = moved && b >= 0;
    const int32_t sa = warp_add(cur_add, a, add);
    const int32_t sb = warp_add(cur_sub, b, sub);
    if (add) {
      add_rows[sa] = (int32_t)i;
      add_lab[sa] = a;
    }
    if (sub) {
      sub_rows[sb] = (int32_t)i;
      sub_lab[sb] = b;
    }
  }
}

__global__ void delta_counts_kernel(const int32_t *__restrict__ hist_add, const int32_t *__restrict__ hist_sub,
                                    int K, int64_t *counts) {
  const int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (k < K) counts[k] += (int64_t)hist_add[k] - (int64_t)hist_sub[k];
}

// J = sum ||x||^2 + sum_k (n_k ||c_k||^2 - 2 c_k . S_k), fp64, with the centres
// that entered this update.  One block per centre; block 0 adds sum ||x||^2.
template <int DT>
__global__ void __launch_bounds__(256) update_objective_kernel(const double *__restrict__ sums,
                                                               const int64_t *__restrict__ counts,
                                                               const float *__restrict__ C, int d,
                                                               const double *__restrict__ x2sum, Header *hdr) {
  __shared__ double part[8];
  const int k = blockIdx.x;
  const double n = (double)counts[k];
  double acc = 0.0;
  if (n > 0.0) {
    for (int j = threadIdx.x; j < d; j += blockDim.x) {
      float c = C[(int64_t)k * d + j];
      if (DT == HME_BF16) c = __bfloat162float(__float2bfloat16_rn(c));
      const double cd = (double)c;
      acc += cd * (n * cd - 2.0 * sums[(int64_t)k * d + j]);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += part[w];
    if (k == 0) t += *x2sum;
    atomicAdd(&hdr->objective, t);
  }
}

__global__ void update_finalize_kernel(const double *__restrict__ sums, const int64_t *__restrict__ hist, int K,
                                       int d, float *__restrict__ C, int64_t *__restrict__ counts_out) {
  // hist: the persistent per-cluster counts
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

// Re-seeding in one pass when at most kReseedFast clusters are empty.  The
// rule takes rows in the order (mind descending, index ascending); with the
// unique 64-bit key (bits of mind, which is >= 0, then the inverted index) that
// order is "key descending", so the E picks are the E largest keys.  Every warp
// keeps its E largest keys (sorted, in shared memory) while streaming mind at
// full bandwidth; one block then merges the sorted lists.  Key 0 is "no row".
constexpr int kReseedFast = 64;
constexpr int kSelWarps = 8;

__device__ __forceinline__ unsigned long long reseed_key(const float *mind, int64_t i) {
  float v = mind ? mind[i] : 0.0f;
  if (!(v >= 0.0f)) v = 0.0f;  // NaN or negative: never above a real distance
  return ((unsigned long long)__float_as_uint(v) << 32) | (unsigned long long)(0xFFFFFFFFu - (uint32_t)i);
}

__device__ __forceinline__ int count_empty(const int64_t *counts, int K) {
  int e = 0;
  for (int k = 0; k < K; ++k) e += counts[k] == 0;
  return e;
}

__global__ void __launch_bounds__(32 * kSelWarps) reseed_select_kernel(const float *__restrict__ mind, int64_t N,
                                                                       const int64_t *__restrict__ counts, int K,
                                                                       unsigned long long *cand) {
  __shared__ unsigned long long lists[kSelWarps][kReseedFast];
  __shared__ int E_s;
  if (threadIdx.x == 0) E_s = count_empty(counts, K);
  __syncthreads();
  const int E = E_s;
  if (E == 0 || E > kReseedFast) return;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  unsigned long long *L = lists[warp];
  for (int j = lane; j < kReseedFast; j += 32) L[j] = 0ull;
  __syncwarp();
  unsigned long long thr = 0ull;  // E-th largest key of this warp so far
  const int64_t gw = (int64_t)blockIdx.x * kSelWarps + warp;
  const int64_t nw = (int64_t)gridDim.x * kSelWarps;
  for (int64_t base = gw * 32; base < N; base += nw * 32) {
    const int64_t i = base + lane;
    const unsigned long long key = i < N ? reseed_key(mind, i) : 0ull;
    unsigned hits = __ballot_sync(0xffffffffu, key > thr);
    while (hits) {
      const int src = __ffs(hits) - 1;
      hits &= hits - 1;
      const unsigned long long k = __shfl_sync(0xffffffffu, key, src);
      if (lane == 0 && k > L[E - 1]) {  // insert into the descending list
        int j = E - 1;
        while (j > 0 && L[j - 1] < k) {
          L[j] = L[j - 1];
          --j;
        }
        L[j] = k;
      }
      __syncwarp();
      thr = L[E - 1];
    }
  }
  for (int j = lane; j < kReseedFast; j += 32) cand[gw * kReseedFast + j] = j < E ? L[j] : 0ull;
}

template <int DT>
__global__ void __launch_bounds__(1024) reseed_apply_kernel(const void *__restrict__ X, int d, int64_t ldx,
                                                            const int64_t *__restrict__ counts, int K,
                                                            const unsigned long long *__restrict__ cand, int nlists,
                                                            float *C, int32_t *n_reseeded) {
  __shared__ int E_s;
  __shared__ unsigned long long best_k[32];
  __shared__ int best_l[32];
  __shared__ unsigned long long pick_key;
  __shared__ int pick_list;
  extern __shared__ int heads[];  // next position in each candidate list
  if (threadIdx.x == 0) E_s = count_empty(counts, K);
  __syncthreads();
  const int E = E_s;
  if (E > kReseedFast) return;  // the general kernel handles it
  if (E == 0) {
    if (threadIdx.x == 0 && n_reseeded) *n_reseeded = 0;
    return;
  }
  for (int l = threadIdx.x; l < nlists; l += blockDim.x) heads[l] = 0;
  __syncthreads();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int taken = 0, kscan = 0;
  for (int r = 0; r < E; ++r) {
    unsigned long long bk = 0ull;
    int bl = -1;
    for (int l = threadIdx.x; l < nlists; l += blockDim.x) {
      const int h = heads[l];
      const unsigned long long k = h < kReseedFast ? cand[(int64_t)l * kReseedFast + h] : 0ull;
      if (k > bk) {
        bk = k;
        bl = l;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const unsigned long long ok = __shfl_xor_sync(0xffffffffu, bk, o);
      const int ol = __shfl_xor_sync(0xffffffffu, bl, o);
      if (ok > bk) {
        bk = ok;
        bl = ol;
      }
    }
    if (lane == 0) {
      best_k[warp] = bk;
      best_l[warp] = bl;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      unsigned long long k = 0ull;
      int l = -1;
      for (int w = 0; w < (int)(blockDim.x >> 5); ++w)
        if (best_k[w] > k) {
          k = best_k[w];
          l = best_l[w];
        }
      pick_key = k;
      pick_list = l;
      if (l >= 0) heads[l] += 1;
    }
    __syncthreads();
    if (pick_key == 0ull) break;  // every row already taken
    // the r-th pick goes to the r-th empty cluster (ascending k)
    while (counts[kscan] != 0) ++kscan;
    const int64_t row = (int64_t)(0xFFFFFFFFu - (uint32_t)(pick_key & 0xFFFFFFFFull));
    for (int j = threadIdx.x; j < d; j += blockDim.x) {
      float x;
      if (DT == HME_BF16)
        x = __bfloat162float(static_cast<const __nv_bfloat16 *>(X)[row * ldx + j]);
      else
        x = static_cast<const float *>(X)[row * ldx + j];
      C[(int64_t)kscan * d + j] = x;
    }
    ++kscan;
    ++taken;
    __syncthreads();
  }
  if (threadIdx.x == 0 && n_reseeded) *n_reseeded = taken;
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
  int n_empty = 0;
  for (int k = threadIdx.x; k < K; k += blockDim.x) n_empty += (hist[k] == 0);
  if (__syncthreads_count(n_empty) <= kReseedFast) return;  // handled by the one-pass selection
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
                 const int64_t *valid_total, double *sums, double *x2sum, float sign, bool device_rows,
                 cudaStream_t s) {
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
  if (!device_rows && nx * min_rows > N) nx = (N + min_rows - 1) / min_rows;
  if (nx < 1) nx = 1;
  const int64_t rpb = device_rows ? 0 : (N + nx - 1) / nx;
  dim3 grid((unsigned)nx, (unsigned)ny);
  update_sums_kernel<DT, VW><<<grid, kUpdThreads, 0, s>>>(X, N, d, ldx, perm, slab, valid_total, V, G, rpb, sums,
                                                          x2sum, sign);
  count_launch();
}

void launch_sums_any(const void *X, int64_t N, int d, int64_t ldx, int dtype, const int32_t *perm,
                     const int32_t *slab, const int64_t *valid_total, double *sums, double *x2sum, float sign,
                     bool device_rows, cudaStream_t s) {
  const bool al = (reinterpret_cast<uintptr_t>(X) & 15u) == 0;
  if (dtype == HME_F32) {
    if (al && d % 4 == 0 && ldx % 4 == 0)
      launch_sums<HME_F32, 4>(X, N, d, ldx, perm, slab, valid_total, sums, x2sum, sign, device_rows, s);
    else
      launch_sums<HME_F32, 1>(X, N, d, ldx, perm, slab, valid_total, sums, x2sum, sign, device_rows, s);
  } else {
    if (al && d % 8 == 0 && ldx % 8 == 0)
      launch_sums<HME_BF16, 8>(X, N, d, ldx, perm, slab, valid_total, sums, x2sum, sign, device_rows, s);
    else
      launch_sums<HME_BF16, 1>(X, N, d, ldx, perm, slab, valid_total, sums, x2sum, sign, device_rows, s);
  }
}

}  // namespace

cudaError_t launch_update(const void *X, int64_t N, int d, int64_t ldx, int dtype, const int32_t *labels,
                          const int32_t *prev_labels, const int32_t *perm, const int32_t *sorted_labels,
                          const int64_t *hist, const int64_t *valid_total, const float *mind, int K,
                          UpdateState st, DeltaScratch ds, float *C, int64_t *counts_out, int32_t *n_reseeded,
                          Header *hdr, cudaStream_t s) {
  cudaError_t e;
  if (!prev_labels) {
    // full pass: recompute the state from scratch
    e = cudaMemsetAsync(st.sums, 0, (size_t)K * d * sizeof(double), s);
    if (e != cudaSuccess) return e;
    e = cudaMemsetAsync(st.x2sum, 0, sizeof(double), s);
    if (e != cudaSuccess) return e;
    e = cudaMemcpyAsync(st.counts, hist, (size_t)K * sizeof(int64_t), cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return e;
    if (N > 0)
      launch_sums_any(X, N, d, ldx, dtype, perm, sorted_labels, valid_total, st.sums, st.x2sum, 1.0f, false, s);
  } else if (N > 0) {
    // incremental: only the rows whose label changed
    e = cudaMemsetAsync(ds.hist_add, 0, (size_t)2 * K * sizeof(int32_t), s);  // hist_add, hist_sub adjacent
    if (e != cudaSuccess) return e;
    int64_t blocks = (int64_t)num_sms() * 8;
    const int64_t want = (N + 255) / 256;
    if (blocks > want) blocks = want;
    delta_count_kernel<<<(unsigned)blocks, 256, 0, s>>>(labels, prev_labels, N, K, ds.hist_add, ds.hist_sub, hdr);
    delta_scan_kernel<<<1, 1024, 0, s>>>(ds.hist_add, ds.hist_sub, K, ds.cur_add, ds.cur_sub, ds.totals);
    delta_report_kernel<<<1, 1, 0, s>>>(ds.totals, hdr);
    count_launch();
    delta_fill_kernel<<<(unsigned)blocks, 256, 0, s>>>(labels, prev_labels, N, K, ds.cur_add, ds.cur_sub,
                                                       ds.add_rows, ds.add_lab, ds.sub_rows, ds.sub_lab);
    count_launch(3);
    launch_sums_any(X, N, d, ldx, dtype, ds.add_rows, ds.add_lab, ds.totals + 0, st.sums, st.x2sum, 1.0f, true, s);
    launch_sums_any(X, N, d, ldx, dtype, ds.sub_rows, ds.sub_lab, ds.totals + 1, st.sums, st.x2sum, -1.0f, true,
                    s);
    delta_counts_kernel<<<(K + 255) / 256, 256, 0, s>>>(ds.hist_add, ds.hist_sub, K, st.counts);
    count_launch();
  }
  if (dtype == HME_F32)
    update_objective_kernel<HME_F32><<<K, 256, 0, s>>>(st.sums, st.counts, C, d, st.x2sum, hdr);
  else
    update_objective_kernel<HME_BF16><<<K, 256, 0, s>>>(st.sums, st.counts, C, d, st.x2sum, hdr);
  const int64_t tot = (int64_t)K * d > K ? (int64_t)K * d : K;
  update_finalize_kernel<<<(unsigned)((tot + 255) / 256), 256, 0, s>>>(st.sums, st.counts, K, d, C, counts_out);
  {
    const int nblk = (num_sms() < kMaxSms ? num_sms() : kMaxSms) * 2;  // the candidate region holds kMaxSms * 2 blocks
    const int nlists = nblk * kSelWarps;
    reseed_select_kernel<<<nblk, 32 * kSelWarps, 0, s>>>(mind, N, st.counts, K, ds.cand);
    const size_t hsm = (size_t)nlists * sizeof(int);
    if (dtype == HME_F32)
      reseed_apply_kernel<HME_F32><<<1, 1024, hsm, s>>>(X, d, ldx, st.counts, K, ds.cand, nlists, C, n_reseeded);
    else
      reseed_apply_kernel<HME_BF16><<<1, 1024, hsm, s>>>(X, d, ldx, st.counts, K, ds.cand, nlists, C, n_reseeded);
  }
  if (dtype == HME_F32)
    update_reseed_kernel<HME_F32><<<1, 1024, 0, s>>>(X, N, d, ldx, mind, st.counts, K, C, n_reseeded);
  else
    update_reseed_kernel<HME_BF16><<<1, 1024, 0, s>>>(X, N, d, ldx, mind, st.counts, K, C, n_reseeded);
  count_launch(5);
  return cudaGetLastError();
}

}  // namespace hme
