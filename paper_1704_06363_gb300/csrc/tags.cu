// tags.cu -- tag statistics of a clustering (Section 4.5, "Analysis of
// YFCC100M clusters"): how often each tag occurs in each cluster (the bars of
// the tag-over-cluster histograms) and, per tag, the sparsity
// ||c(t)||_1 / ||c(t)||_2 of its distribution c(t) over the clusters (the x
// axis of the sparsity-versus-accuracy figure).
//
// Input is the partitioned form that hme_partition writes: cluster k owns the
// points offsets[k] .. offsets[k+1]-1 and therefore the contiguous tag range
// tag_off[offsets[k]] .. tag_off[offsets[k+1]]-1.  So one cluster's counts are
// a histogram of one contiguous id range:
//   tag_chunks    one block: every cluster's range is cut into chunks of at
//                 most kTagChunk tags (an empty cluster is one empty chunk);
//                 exclusive scan of the chunk counts;
//   tag_zero      rows of clusters with several chunks start at zero (they are
//                 accumulated with atomics);
//   tag_hist      persistent blocks over the chunks: a shared-memory histogram
//                 of the V tag ids (equal ids of a warp add once, with
//                 __match_any_sync), then the row of counts goes out with
//                 plain stores when the cluster is one chunk, or 64-bit
//                 atomics of the non-zero bins otherwise.  A vocabulary
//                 too large for shared memory counts straight into the
//                 (zeroed) global rows with the same warp aggregation;
//   tag_sparsity  a block per 32 tags, its warps splitting the clusters
//                 (reads coalesced over tags): l1 and sum of squares in fp64
//                 (exact for integer counts below 2^53), ratio; 0 for absent
//                 tags.
// Tags outside [0, V) are skipped and set kStatusBadTag.
#include "hme_common.cuh"

namespace hme {

namespace {

constexpr int64_t kTagChunk = 65536;
constexpr int kTagThreads = 512;

__global__ void __launch_bounds__(1024) tag_chunks_kernel(const int64_t *__restrict__ offsets,
                                                          const int64_t *__restrict__ tag_off, int K,
                                                          int64_t *chunk_start, Header *hdr) {
  __shared__ int64_t wsum[32];
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const int per = (K + 1023) / 1024;
  const int k0 = t * per, k1 = min(K, k0 + per);
  auto chunks_of = [&](int k) -> int64_t {
    const int64_t a = tag_off[offsets[k]], b = tag_off[offsets[k + 1]];
    if (b < a) {
      atomicOr(&hdr->status, (uint32_t)kStatusBadTag);
      return 1;
    }
    const int64_t n = (b - a + kTagChunk - 1) / kTagChunk;
    return n > 0 ? n : 1;
  };
  int64_t local = 0;
  for (int k = k0; k < k1; ++k) local += chunks_of(k);
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
    chunk_start[k] = run;
    run += chunks_of(k);
  }
  if (t == 1023) chunk_start[K] = run;
}

// Zero the rows that are accumulated with atomics: clusters of several chunks,
// or every row when the histogram lives in global memory (all_rows).
__global__ void tag_zero_kernel(const int64_t *__restrict__ chunk_start, int K, int V, bool all_rows,
                                int64_t *counts) {
  for (int k = blockIdx.x; k < K; k += gridDim.x) {
    if (!all_rows && chunk_start[k + 1] - chunk_start[k] <= 1) continue;
    int64_t *row = counts + (int64_t)k * V;
    for (int t = threadIdx.x; t < V; t += blockDim.x) row[t] = 0;
  }
}

// Cluster of chunk c: the last k with chunk_start[k] <= c.
__device__ __forceinline__ int chunk_cluster(const int64_t *chunk_start, int K, int64_t c) {
  int lo = 0, hi = K;  // chunk_start[lo] <= c < chunk_start[hi]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (chunk_start[mid] <= c)
      lo = mid;
    else
      hi = mid;
  }
  return lo;
}

template <bool SMEM>
__global__ void __launch_bounds__(kTagThreads) tag_hist_kernel(const int64_t *__restrict__ offsets,
                                                               const int64_t *__restrict__ tag_off,
                                                               const int32_t *__restrict__ tags, int K, int V,
                                                               const int64_t *__restrict__ chunk_start,
                                                               int64_t *counts, Header *hdr) {
  extern __shared__ int32_t hist[];  // V counters (SMEM)
  __shared__ int k_s;
  const int lane = threadIdx.x & 31;
  const int64_t nchunks = chunk_start[K];
  bool bad = false;
  for (int64_t c = blockIdx.x; c < nchunks; c += gridDim.x) {
    if (threadIdx.x == 0) k_s = chunk_cluster(chunk_start, K, c);
    if (SMEM)
      for (int t = threadIdx.x; t < V; t += blockDim.x) hist[t] = 0;
    __syncthreads();
    const int k = k_s;
    const int64_t j = c - chunk_start[k];
    const int64_t nk = chunk_start[k + 1] - chunk_start[k];
    const int64_t a = tag_off[offsets[k]], b = tag_off[offsets[k + 1]];
    const int64_t lo = a + j * kTagChunk;
    const int64_t hi = b < lo + kTagChunk ? b : lo + kTagChunk;
    int64_t *row = counts + (int64_t)k * V;
    // whole warps step together so that __match_any_sync sees every lane
    for (int64_t base = lo + (threadIdx.x & ~31); base < hi; base += blockDim.x) {
      const int64_t i = base + lane;
      const int32_t t = i < hi ? __ldg(tags + i) : -1;
      const bool valid = i < hi && t >= 0 && t < V;
      if (i < hi && !valid) bad = true;
      const unsigned act = __ballot_sync(0xffffffffu, valid);
      const unsigned peers = __match_any_sync(0xffffffffu, valid ? t : -1) & act;
      if (valid && lane == __ffs(peers) - 1) {
        if (SMEM)
          atomicAdd(&hist[t], (int32_t)__popc(peers));
        else
          atomicAdd(reinterpret_cast<unsigned long long *>(row + t), (unsigned long long)__popc(peers));
      }
    }
    __syncthreads();
    if (SMEM) {
      if (nk == 1) {
        for (int t = threadIdx.x; t < V; t += blockDim.x) row[t] = hist[t];
      } else {
        for (int t = threadIdx.x; t < V; t += blockDim.x)
          if (hist[t] != 0) atomicAdd(reinterpret_cast<unsigned long long *>(row + t), (unsigned long long)hist[t]);
      }
      __syncthreads();  // hist is cleared for the next chunk
    }
  }
  if (bad) atomicOr(&hdr->status, (uint32_t)kStatusBadTag);
}

// One block per 32 consecutive tags (lane = tag, coalesced 256-byte reads of a
// row segment); its 8 warps take every 8th cluster and combine in shared memory.
constexpr int kSpWarps = 8;

__global__ void __launch_bounds__(32 * kSpWarps) tag_sparsity_kernel(const int64_t *__restrict__ counts, int K, int V,
                                                                     double *sparsity) {
  __shared__ double part[2][kSpWarps][32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int t = blockIdx.x * 32 + lane;
  double l1 = 0.0, l2sq = 0.0;
  if (t < V) {
#pragma unroll 8
    for (int k = warp; k < K; k += kSpWarps) {
      const double c = (double)__ldg(counts + (int64_t)k * V + t);
      l1 += c;
      l2sq = fma(c, c, l2sq);
    }
  }
  part[0][warp][lane] = l1;
  part[1][warp][lane] = l2sq;
  __syncthreads();
  if (warp == 0 && t < V) {
    double a = 0.0, b = 0.0;
    for (int w = 0; w < kSpWarps; ++w) {  // counts are integers below 2^53: every partial sum is exact
      a += part[0][w][lane];
      b += part[1][w][lane];
    }
    sparsity[t] = a > 0.0 ? a / sqrt(b) : 0.0;
  }
}

}  // namespace

size_t tag_hist_smem_limit() { return (size_t)200 * 1024; }

cudaError_t launch_tag_hist(const int64_t *offsets, const int64_t *tag_off, const int32_t *tags, int K, int V,
                            int64_t *chunk_start, int64_t *counts, double *sparsity, Header *hdr, cudaStream_t s) {
  tag_chunks_kernel<<<1, 1024, 0, s>>>(offsets, tag_off, K, chunk_start, hdr);
  const size_t smem = (size_t)V * sizeof(int32_t);
  const bool in_smem = smem <= tag_hist_smem_limit();
  const int zb = K < 1024 ? K : 1024;
  tag_zero_kernel<<<zb, 256, 0, s>>>(chunk_start, K, V, !in_smem, counts);
  int grid = num_sms();
  cudaError_t e;
  if (in_smem) {
    e = cudaFuncSetAttribute(tag_hist_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int per_sm = (int)((size_t)(227 * 1024) / (smem + 1024));
    grid *= per_sm < 1 ? 1 : (per_sm > 4 ? 4 : per_sm);
    tag_hist_kernel<true><<<grid, kTagThreads, smem, s>>>(offsets, tag_off, tags, K, V, chunk_start, counts, hdr);
  } else {
    grid *= 4;
    tag_hist_kernel<false><<<grid, kTagThreads, 0, s>>>(offsets, tag_off, tags, K, V, chunk_start, counts, hdr);
  }
  count_launch(3);
  if (sparsity) {
    tag_sparsity_kernel<<<(V + 31) / 32, 32 * kSpWarps, 0, s>>>(counts, K, V, sparsity);
    count_launch();
  }
  return cudaGetLastError();
}

}  // namespace hme
