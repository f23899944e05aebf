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
// Then, in one kernel:
//   objective   J = sum ||x||^2 - 2 sum_k c_k . S_k + sum_k n_k ||c_k||^2 in
//               fp64 with the centres that entered this update (bf16-rounded
//               for bf16 features): the Lloyd objective of (C_t, labels).
//   finalize    c_k = S_k * (1 / n_k) in fp64 (within 2^-52 relative of the
//               quotient; one divide per centre), rounded once to fp32, for
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
// Rows come from one list (perm, slab; *n1 entries, added) followed by an
// optional second list (perm2, slab2; *n2 entries, subtracted).  With
// rows_per_block == 0 the split is made on the device, at least kMinRows rows
// per block so that a short list does not turn into one flush per row.
constexpr int64_t kMinRows = 16;

template <int DT, int VW>
__global__ void __launch_bounds__(kUpdThreads) update_sums_kernel(const void *__restrict__ X, int64_t N, int d,
                                                                  int64_t ldx, const int32_t *__restrict__ perm,
                                                                  const int32_t *__restrict__ slab,
                                                                  const int64_t *__restrict__ n1,
                                                                  const int32_t *__restrict__ perm2,
                                                                  const int32_t *__restrict__ slab2,
                                                                  const int64_t *__restrict__ n2, int V, int G,
                                                                  int64_t rows_per_block, double *sums,
                                                                  double *x2sum) {
  __shared__ double qpart[kUpdThreads / 32];
  const int g = threadIdx.x / V;
  const int t = threadIdx.x - g * V;
  const int vcol = blockIdx.y * V + t;
  const int col = vcol * VW;
  const int64_t na = min(N, *n1);
  const int64_t nrows = na + (n2 ? min(N, *n2) : 0);
  int64_t rpb = rows_per_block;
  if (rpb <= 0) rpb = max(kMinRows, (nrows + gridDim.x - 1) / gridDim.x);
  const int64_t b0 = (int64_t)blockIdx.x * rpb;
  const int64_t b1 = min(nrows, b0 + rpb);
  const int64_t per = (b1 - b0 + G - 1) / G;
  const int64_t r0 = b0 + g * per;
  const int64_t r1 = min(b1, r0 + per);
  const bool active = (g < G) && (col < d) && (r0 < r1);
  double qd = 0.0;
  // entry j of the joined list: its row and its key (label, or ~label when subtracted)
  auto entry = [&](int64_t j, int &key) -> int64_t {
    if (j < na) {
      key = __ldg(slab + j);
      return __ldg(perm + j);
    }
    key = ~__ldg(slab2 + (j - na));
    return __ldg(perm2 + (j - na));
  };

  if (active) {
    float acc[VW];
    double accd[VW];
    float q = 0.0f;
    int cur;
    entry(r0, cur);
    auto fold = [&]() {
#pragma unroll
      for (int e = 0; e < VW; ++e) {
        accd[e] += (double)acc[e];
        acc[e] = 0.0f;
      }
      qd += (double)q;
      q = 0.0f;
    };
    auto flush = [&](int key) {
      fold();
      double *dst = sums + (int64_t)(key >= 0 ? key : ~key) * d + col;
#pragma unroll
      for (int e = 0; e < VW; ++e) {
        if (VW == 1 || col + e < d) atomicAdd(dst + e, accd[e]);
        accd[e] = 0.0;
      }
    };
    auto add_row = [&](const float (&v)[VW], int key) {
      const float sg = key >= 0 ? 1.0f : -1.0f;
#pragma unroll
      for (int e = 0; e < VW; ++e) {
        acc[e] += sg * v[e];
        q = fmaf(sg * v[e], v[e], q);
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
      int key[kUnroll];
      float v[kUnroll][VW];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int64_t row = entry(j + u, key[u]);
        Vec<DT, VW>::load(X, row * ldx + col, v[u]);
      }
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        if (key[u] != cur) {
          flush(cur);
          cur = key[u];
        }
        add_row(v[u], key[u]);
      }
      if ((since += kUnroll) >= 64) {
        fold();
        since = 0;
      }
    }
    for (; j < r1; ++j) {
      int key;
      const int64_t row = entry(j, key);
      float v[VW];
      Vec<DT, VW>::load(X, row * ldx + col, v);
      if (key != cur) {
        flush(cur);
        cur = key;
      }
      add_row(v, key);
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

// Incremental update, in three small kernels over the label vectors:
//   delta_count  the rows are cut into ntiles contiguous tiles, one block
//                each; a block counts its rows whose label changed per new
//                label (to add) and per old label (to subtract) in shared
//                memory (labels outside [0, K) count as unassigned on either
//                side) and writes its row of the ntiles x 2K count matrix;
//   delta_colscan for each of the 2K counts, the exclusive prefix over the
//                tiles and the total (hist_add, hist_sub);
//   delta_scan   exclusive prefix of both totals -> the lists' bucket starts
//                and the list lengths; also moves n_k by (added - subtracted);
//   delta_fill   a block takes slots from shared cursors (bucket start +
//                earlier tiles' rows of the bucket): the changed rows grouped
//                by label (order inside a group is irrelevant for sums), as
//                (row, label) lists;
// then one sums launch runs over both lists (added, then subtracted).
constexpr int kDeltaThreads = 512;
constexpr int64_t kDeltaTile = 16384;  // rows per tile at least (tiles: at most kDeltaTiles)
constexpr int kDeltaTiles = 304;

// Labels i .. i+VEC-1 of both vectors (16-byte loads when VEC == 4); entries
// past N read as -1 on both sides (unchanged).
template <int VEC>
__device__ __forceinline__ void load_pair(const int32_t *labels, const int32_t *prev, int64_t i, int64_t N,
                                          int (&a)[VEC], int (&b)[VEC]) {
  if (VEC == 4 && i + 4 <= N) {
    const int4 x = __ldg(reinterpret_cast<const int4 *>(labels + i));
    const int4 y = __ldg(reinterpret_cast<const int4 *>(prev + i));
    a[0] = x.x, a[1] = x.y, a[2] = x.z, a[3] = x.w;
    b[0] = y.x, b[1] = y.y, b[2] = y.z, b[3] = y.w;
  } else {
#pragma unroll
    for (int e = 0; e < VEC; ++e) {
      a[e] = i + e < N ? __ldg(labels + i + e) : -1;
      b[e] = i + e < N ? __ldg(prev + i + e) : -1;
    }
  }
}

template <int VEC>
__global__ void __launch_bounds__(kDeltaThreads) delta_count_kernel(const int32_t *__restrict__ labels,
                                                                    const int32_t *__restrict__ prev, int64_t N,
                                                                    int K, int64_t tile, int32_t *__restrict__ mat,
                                                                    Header *hdr) {
  extern __shared__ int32_t dh[];  // [0, K): to add; [K, 2K): to subtract
  for (int k = threadIdx.x; k < 2 * K; k += kDeltaThreads) dh[k] = 0;
  __syncthreads();
  const int64_t t0 = (int64_t)blockIdx.x * tile, t1 = min(N, t0 + tile);
  bool bad = false;
  for (int64_t i = t0 + (int64_t)threadIdx.x * VEC; i < t1; i += (int64_t)kDeltaThreads * VEC) {
    int a[VEC], b[VEC];
    load_pair<VEC>(labels, prev, i, t1, a, b);
#pragma unroll
    for (int e = 0; e < VEC; ++e) {
      if (i + e < t1 && (a[e] < 0 || a[e] >= K)) bad = true;
      const int na = (a[e] >= 0 && a[e] < K) ? a[e] : -1;
      const int nb = (b[e] >= 0 && b[e] < K) ? b[e] : -1;
      if (na != nb) {
        if (na >= 0) atomicAdd(&dh[na], 1);
        if (nb >= 0) atomicAdd(&dh[K + nb], 1);
      }
    }
  }
  if (bad) atomicOr(&hdr->status, (uint32_t)kStatusBadLabel);
  __syncthreads();
  int32_t *row = mat + (int64_t)blockIdx.x * 2 * K;
  for (int k = threadIdx.x; k < 2 * K; k += kDeltaThreads) row[k] = dh[k];
}

// For every column c of the ntiles x 2K count matrix: the exclusive prefix
// over the tiles in place, the column total to hist[c] (hist_add then
// hist_sub, adjacent).  A block takes 32 columns: warp w sums its strip of
// about ntiles / 32 tiles (lane = column), one warp scans the 32 strip sums,
// then every warp rewrites its strip from its strip's start.
__global__ void __launch_bounds__(1024) delta_colscan_kernel(int32_t *__restrict__ mat, int64_t ntiles, int K,
                                                             int32_t *__restrict__ hist) {
  __shared__ int32_t part[32][33];
  const int W = 2 * K;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  const int c = blockIdx.x * 32 + tx;
  const int64_t R = (ntiles + 31) / 32;
  const int64_t r0 = ty * R, r1 = min(ntiles, r0 + R);
  int32_t sum = 0;
  if (c < W)
    for (int64_t t = r0; t < r1; ++t) sum += mat[t * W + c];
  part[ty][tx] = sum;
  __syncthreads();
  if (ty == 0) {
    int32_t run = 0;
    for (int g = 0; g < 32; ++g) {
      const int32_t v = part[g][tx];
      part[g][tx] = run;
      run += v;
    }
    if (c < W) hist[c] = run;
  }
  __syncthreads();
  if (c < W) {
    int32_t run = part[ty][tx];
    for (int64_t t = r0; t < r1; ++t) {
      const int32_t v = mat[t * W + c];
      mat[t * W + c] = run;
      run += v;
    }
  }
}

// Exclusive prefix of hist_add and hist_sub (one block), the fill cursors,
// totals = {rows to add, rows to subtract}, the moved-row count in the header
// and n_k += added_k - subtracted_k.
__global__ void __launch_bounds__(1024) delta_scan_kernel(const int32_t *__restrict__ hist_add,
                                                          const int32_t *__restrict__ hist_sub, int K,
                                                          int32_t *cur_add, int32_t *cur_sub, int64_t *totals,
                                                          int64_t *counts, Header *hdr) {
  __shared__ int64_t wsum[32];
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const int per = (K + 1023) / 1024;
  const int k0 = t * per, k1 = min(K, k0 + per);
  for (int which = 0; which < 2; ++which) {
    const int32_t *h = which == 0 ? hist_add : hist_sub;
    int32_t *cur = which == 0 ? cur_add : cur_sub;
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
    if (t == 1023) {
      totals[which] = run;
      if (which == 0) hdr->moved_rows = (uint32_t)min(run, (int64_t)0xFFFFFFFF);
    }
    __syncthreads();
  }
  for (int k = t; k < K; k += blockDim.x) counts[k] += (int64_t)hist_add[k] - (int64_t)hist_sub[k];
}

template <int VEC>
__global__ void __launch_bounds__(kDeltaThreads) delta_fill_kernel(const int32_t *__restrict__ labels,
                                                                   const int32_t *__restrict__ prev, int64_t N,
                                                                   int K, int64_t tile,
                                                                   const int32_t *__restrict__ mat,
                                                                   const int32_t *__restrict__ cur_add,
                                                                   const int32_t *__restrict__ cur_sub,
                                                                   int32_t *add_rows, int32_t *add_lab,
                                                                   int32_t *sub_rows, int32_t *sub_lab) {
  extern __shared__ int32_t dc[];  // this tile's next slot of each list bucket: [0, K) add, [K, 2K) subtract
  const int32_t *row = mat + (int64_t)blockIdx.x * 2 * K;
  for (int k = threadIdx.x; k < K; k += kDeltaThreads) {
    dc[k] = cur_add[k] + row[k];
    dc[K + k] = cur_sub[k] + row[K + k];
  }
  __syncthreads();
  const int64_t t0 = (int64_t)blockIdx.x * tile, t1 = min(N, t0 + tile);
  for (int64_t i = t0 + (int64_t)threadIdx.x * VEC; i < t1; i += (int64_t)kDeltaThreads * VEC) {
    int a[VEC], b[VEC];
    load_pair<VEC>(labels, prev, i, t1, a, b);
#pragma unroll
    for (int e = 0; e < VEC; ++e) {
      const int na = (a[e] >= 0 && a[e] < K) ? a[e] : -1;
      const int nb = (b[e] >= 0 && b[e] < K) ? b[e] : -1;
      if (na != nb) {
        if (na >= 0) {
          const int32_t sa = atomicAdd(&dc[na], 1);
          add_rows[sa] = (int32_t)(i + e);
          add_lab[sa] = na;
        }
        if (nb >= 0) {
          const int32_t sb = atomicAdd(&dc[K + nb], 1);
          sub_rows[sb] = (int32_t)(i + e);
          sub_lab[sb] = nb;
        }
      }
    }
  }
}

// Objective and new centres in one pass over (S, n, C); one block per
// (centre k, 1024-column slice):
//   J = sum ||x||^2 + sum_k (n_k ||c_k||^2 - 2 c_k . S_k) in fp64 with the
//       centres that entered this update (bf16-rounded for bf16 features);
//       block (0, 0) adds sum ||x||^2;
//   c_k = S_k * (1 / n_k) in fp64, rounded once to fp32, for non-empty k (each
//       element is read, for J, by the thread that then overwrites it);
//   counts_out = n.
constexpr int kFinThreads = 256, kFinPer = 4;

template <int DT>
__global__ void __launch_bounds__(kFinThreads) update_finish_kernel(const double *__restrict__ sums,
                                                                    const int64_t *__restrict__ counts, float *C,
                                                                    int d, const double *__restrict__ x2sum,
                                                                    int64_t *counts_out, Header *hdr) {
  __shared__ double part[kFinThreads / 32];
  const int k = blockIdx.x;
  const int64_t nk = counts[k];
  const double n = (double)nk;
  const double inv = nk > 0 ? 1.0 / n : 0.0;
  double acc = 0.0;
  if (nk > 0) {
#pragma unroll
    for (int u = 0; u < kFinPer; ++u) {
      const int j = blockIdx.y * (kFinThreads * kFinPer) + u * kFinThreads + threadIdx.x;
      if (j < d) {
        const int64_t at = (int64_t)k * d + j;
        float c = C[at];
        const double S = sums[at];
        if (DT == HME_BF16) c = __bfloat162float(__float2bfloat16_rn(c));
        const double cd = (double)c;
        acc += cd * (n * cd - 2.0 * S);
        C[at] = (float)(S * inv);
      }
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int w = 0; w < kFinThreads / 32; ++w) t += part[w];
    if (k == 0 && blockIdx.y == 0) t += *x2sum;
    if (t != 0.0) atomicAdd(&hdr->objective, t);
    if (counts_out && blockIdx.y == 0) counts_out[k] = nk;
  }
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

// Number of empty clusters, counted by the whole block (every thread must call
// it; blockDim a multiple of 32); *acc is a shared-memory int it may overwrite.
__device__ __forceinline__ int block_count_empty(const int64_t *counts, int K, int *acc) {
  if (threadIdx.x == 0) *acc = 0;
  __syncthreads();
  int e = 0;
  for (int k = threadIdx.x; k < K; k += blockDim.x) e += counts[k] == 0;
  e = __reduce_add_sync(0xffffffffu, e);
  if ((threadIdx.x & 31) == 0 && e != 0) atomicAdd(acc, e);
  __syncthreads();
  return *acc;
}

__global__ void __launch_bounds__(32 * kSelWarps) reseed_select_kernel(const float *__restrict__ mind, int64_t N,
                                                                       const int64_t *__restrict__ counts, int K,
                                                                       unsigned long long *cand) {
  __shared__ unsigned long long lists[kSelWarps][kReseedFast];
  __shared__ int E_s;
  const int E = block_count_empty(counts, K, &E_s);
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
  const int E = block_count_empty(counts, K, &E_s);
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

// List (perm, slab; *n1 rows, added) then optionally (perm2, slab2; *n2 rows,
// subtracted).  device_rows: the row counts are known only on the device.
struct SumsLists {
  const int32_t *perm, *slab;
  const int64_t *n1;
  const int32_t *perm2, *slab2;
  const int64_t *n2;
};

template <int DT, int VW>
void launch_sums(const void *X, int64_t N, int d, int64_t ldx, const SumsLists &l, double *sums, double *x2sum,
                 bool device_rows, cudaStream_t s) {
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
  update_sums_kernel<DT, VW><<<grid, kUpdThreads, 0, s>>>(X, N, d, ldx, l.perm, l.slab, l.n1, l.perm2, l.slab2,
                                                          l.n2, V, G, rpb, sums, x2sum);
  count_launch();
}

void launch_sums_any(const void *X, int64_t N, int d, int64_t ldx, int dtype, const SumsLists &l, double *sums,
                     double *x2sum, bool device_rows, cudaStream_t s) {
  const bool al = (reinterpret_cast<uintptr_t>(X) & 15u) == 0;
  if (dtype == HME_F32) {
    if (al && d % 4 == 0 && ldx % 4 == 0)
      launch_sums<HME_F32, 4>(X, N, d, ldx, l, sums, x2sum, device_rows, s);
    else
      launch_sums<HME_F32, 1>(X, N, d, ldx, l, sums, x2sum, device_rows, s);
  } else {
    if (al && d % 8 == 0 && ldx % 8 == 0)
      launch_sums<HME_BF16, 8>(X, N, d, ldx, l, sums, x2sum, device_rows, s);
    else
      launch_sums<HME_BF16, 1>(X, N, d, ldx, l, sums, x2sum, device_rows, s);
  }
}

__global__ void counts_add_kernel(const int64_t *__restrict__ hist, int K, int64_t *counts) {
  const int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (k < K) counts[k] += hist[k];
}

}  // namespace

// After the sums: objective and new centres, then the re-seed of empty
// clusters from the rows (X may be any device-accessible pointer, e.g.
// page-locked host memory: only the picked rows are read).
cudaError_t launch_update_finish(const void *X, int64_t N, int d, int64_t ldx, int dtype, const float *mind, int K,
                                 UpdateState st, DeltaScratch ds, float *C, int64_t *counts_out, int32_t *n_reseeded,
                                 Header *hdr, cudaStream_t s) {
  {
    const dim3 grid((unsigned)K, (unsigned)((d + kFinThreads * kFinPer - 1) / (kFinThreads * kFinPer)));
    if (dtype == HME_F32)
      update_finish_kernel<HME_F32><<<grid, kFinThreads, 0, s>>>(st.sums, st.counts, C, d, st.x2sum, counts_out, hdr);
    else
      update_finish_kernel<HME_BF16><<<grid, kFinThreads, 0, s>>>(st.sums, st.counts, C, d, st.x2sum, counts_out,
                                                                  hdr);
  }
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
  count_launch(4);
  return cudaGetLastError();
}

// Streamed full pass: add one chunk's rows (sorted by label: perm / sorted
// labels / hist of the chunk) to the state; reset first when asked.
cudaError_t launch_update_add(const void *X, int64_t n, int d, int64_t ldx, int dtype, const int32_t *perm,
                              const int32_t *sorted_labels, const int64_t *hist, const int64_t *valid_total, int K,
                              UpdateState st, bool reset, cudaStream_t s) {
  cudaError_t e;
  if (reset) {
    e = cudaMemsetAsync(st.sums, 0, (size_t)K * d * sizeof(double), s);
    if (e != cudaSuccess) return e;
    e = cudaMemsetAsync(st.x2sum, 0, sizeof(double), s);
    if (e != cudaSuccess) return e;
    e = cudaMemsetAsync(st.counts, 0, (size_t)K * sizeof(int64_t), s);
    if (e != cudaSuccess) return e;
  }
  if (n <= 0) return cudaSuccess;
  counts_add_kernel<<<(K + 255) / 256, 256, 0, s>>>(hist, K, st.counts);
  count_launch();
  launch_sums_any(X, n, d, ldx, dtype, SumsLists{perm, sorted_labels, valid_total, nullptr, nullptr, nullptr},
                  st.sums, st.x2sum, false, s);
  return cudaGetLastError();
}

// Rows per tile of the incremental update: at most kDeltaTiles tiles of at
// least kDeltaTile rows, a multiple of 4 (tiles start on 16-byte boundaries of
// aligned labels).
int64_t delta_tile_len(int64_t N) {
  int64_t tile = (N + kDeltaTiles - 1) / kDeltaTiles;
  if (tile < kDeltaTile) tile = kDeltaTile;
  return (tile + 3) / 4 * 4;
}

int64_t delta_tiles(int64_t N) { return N > 0 ? (N + delta_tile_len(N) - 1) / delta_tile_len(N) : 1; }

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
      launch_sums_any(X, N, d, ldx, dtype, SumsLists{perm, sorted_labels, valid_total, nullptr, nullptr, nullptr},
                    st.sums, st.x2sum, false, s);
  } else if (N > 0) {
    // incremental: only the rows whose label changed
    const int64_t tile = delta_tile_len(N);
    const int64_t ntiles = (N + tile - 1) / tile;
    const bool vec = (reinterpret_cast<uintptr_t>(labels) & 15u) == 0 &&
                     (reinterpret_cast<uintptr_t>(prev_labels) & 15u) == 0;
    const size_t smem = (size_t)2 * K * sizeof(int32_t);
    auto count = vec ? delta_count_kernel<4> : delta_count_kernel<1>;
    auto fill = vec ? delta_fill_kernel<4> : delta_fill_kernel<1>;
    if (smem > 48 * 1024) {
      e = cudaFuncSetAttribute(count, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (e != cudaSuccess) return e;
      e = cudaFuncSetAttribute(fill, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (e != cudaSuccess) return e;
    }
    count<<<(unsigned)ntiles, kDeltaThreads, smem, s>>>(labels, prev_labels, N, K, tile, ds.mat, hdr);
    delta_colscan_kernel<<<(unsigned)((2 * K + 31) / 32), 1024, 0, s>>>(ds.mat, ntiles, K, ds.hist_add);
    delta_scan_kernel<<<1, 1024, 0, s>>>(ds.hist_add, ds.hist_sub, K, ds.cur_add, ds.cur_sub, ds.totals, st.counts,
                                         hdr);
    fill<<<(unsigned)ntiles, kDeltaThreads, smem, s>>>(labels, prev_labels, N, K, tile, ds.mat, ds.cur_add,
                                                        ds.cur_sub, ds.add_rows, ds.add_lab, ds.sub_rows,
                                                        ds.sub_lab);
    count_launch(4);
    launch_sums_any(X, N, d, ldx, dtype,
                    SumsLists{ds.add_rows, ds.add_lab, ds.totals + 0, ds.sub_rows, ds.sub_lab, ds.totals + 1},
                    st.sums, st.x2sum, true, s);
  }
  return launch_update_finish(X, N, d, ldx, dtype, mind, K, st, ds, C, counts_out, n_reseeded, hdr, s);
}

}  // namespace hme
