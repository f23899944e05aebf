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
//                 of the V tag ids in 16-bit fields (one shared atomic per
//                 tag), then the row of counts goes out with
//                 plain stores when the cluster is one chunk, or 64-bit
//                 atomics of the non-zero bins otherwise.  A vocabulary
//                 too large for shared memory counts straight into the
//                 (zeroed) global rows with 64-bit atomics;
//   tag_colsum    blocks of 256 tags x one of 16 slices of the clusters write
//                 each tag's partial l1 and sum of squares (64-bit integers,
//                 exact);
//   tag_sparsity  adds the slices and forms the ratio; 0 for absent tags.
// Tags outside [0, V) are skipped and set kStatusBadTag.
#include "hme_common.cuh"

namespace hme {

namespace {

// at most 65535 tags per chunk: a tag's count in a chunk fits a 16-bit field
constexpr int64_t kTagChunk = 65535;
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

// Shared-memory counters are 16-bit fields, two per 32-bit word (tag t in
// word t / 2, bits 16 (t % 2) ..): a chunk holds at most 65535 tags, so no
// field carries into its neighbour, and twice as many blocks fit an SM.
template <bool SMEM>
__global__ void __launch_bounds__(kTagThreads) tag_hist_kernel(const int64_t *__restrict__ offsets,
                                                               const int64_t *__restrict__ tag_off,
                                                               const int32_t *__restrict__ tags, int K, int V,
                                                               const int64_t *__restrict__ chunk_start,
                                                               int64_t *counts, Header *hdr) {
  extern __shared__ uint32_t hist[];  // (V + 1) / 2 words (SMEM)
  __shared__ int k_s;
  const int lane = threadIdx.x & 31;
  const int words = (V + 1) >> 1;
  const int64_t nchunks = chunk_start[K];
  bool bad = false;
  for (int64_t c = blockIdx.x; c < nchunks; c += gridDim.x) {
    if (threadIdx.x == 0) k_s = chunk_cluster(chunk_start, K, c);
    if (SMEM)
      for (int w = threadIdx.x; w < words; w += blockDim.x) hist[w] = 0u;
    __syncthreads();
    const int k = k_s;
    const int64_t j = c - chunk_start[k];
    const int64_t nk = chunk_start[k + 1] - chunk_start[k];
    const int64_t a = tag_off[offsets[k]], b = tag_off[offsets[k + 1]];
    const int64_t lo = a + j * kTagChunk;
    const int64_t hi = b < lo + kTagChunk ? b : lo + kTagChunk;
    int64_t *row = counts + (int64_t)k * V;
    // 4 loads per thread in flight, then one shared-memory atomic per tag
    // (equal tags of a warp are serialised by the hardware; cheaper than
    // grouping them first)
    for (int64_t base = lo + threadIdx.x; base < hi; base += (int64_t)blockDim.x * 4) {
      int32_t tv[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int64_t i = base + (int64_t)u * blockDim.x;
        tv[u] = i < hi ? __ldg(tags + i) : -1;
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int64_t i = base + (int64_t)u * blockDim.x;
        if (i >= hi) continue;
        const int32_t t = tv[u];
        if (t < 0 || t >= V) {
          bad = true;
          continue;
        }
        if (SMEM)
          atomicAdd(&hist[t >> 1], 1u << (16 * (t & 1)));
        else
          atomicAdd(reinterpret_cast<unsigned long long *>(row + t), 1ull);
      }
    }
    __syncthreads();
    if (SMEM) {
      for (int t = threadIdx.x; t < V; t += blockDim.x) {
        const uint32_t v = (hist[t >> 1] >> (16 * (t & 1))) & 0xFFFFu;
        if (nk == 1)
          row[t] = v;
        else if (v != 0)
          atomicAdd(reinterpret_cast<unsigned long long *>(row + t), (unsigned long long)v);
      }
      __syncthreads();  // hist is cleared for the next chunk
    }
  }
  if (bad) atomicOr(&hdr->status, (uint32_t)kStatusBadTag);
}

// Per-tag l1 and sum of squares over the clusters: a block takes 256
// consecutive tags (2 KB of every row it reads, coalesced) and one of
// kTagSlices slices of the clusters, and writes its partial sums to
// part[slice][0 .. V) and part[slice][V .. 2V); tag_sparsity adds the slices.
// The sums are kept in 64-bit integers (exact: a tag's squared counts add up
// to at most (number of tags)^2 < 2^62), so no per-element fp64 arithmetic is
// needed and the result does not depend on the order; the ratio is formed
// once per tag in fp64.
__global__ void __launch_bounds__(256) tag_colsum_kernel(const int64_t *__restrict__ counts, int K, int V,
                                                         int rows_per_slice, uint64_t *part) {
  const int t = blockIdx.x * 256 + threadIdx.x;
  const int k0 = blockIdx.y * rows_per_slice;
  const int k1 = min(K, k0 + rows_per_slice);
  if (t >= V) return;
  uint64_t l1 = 0, l2sq = 0;
#pragma unroll 8
  for (int k = k0; k < k1; ++k) {
    const uint64_t c = (uint64_t)__ldg(counts + (int64_t)k * V + t);
    l1 += c;
    l2sq += c * c;
  }
  uint64_t *dst = part + (int64_t)blockIdx.y * 2 * V;
  dst[t] = l1;
  dst[V + t] = l2sq;
}

__global__ void __launch_bounds__(256) tag_sparsity_kernel(const uint64_t *__restrict__ part, int V, int slices,
                                                           double *sparsity) {
  const int t = blockIdx.x * 256 + threadIdx.x;
  if (t >= V) return;
  uint64_t l1 = 0, l2sq = 0;
  for (int sl = 0; sl < slices; ++sl) {
    l1 += part[(int64_t)sl * 2 * V + t];
    l2sq += part[(int64_t)sl * 2 * V + V + t];
  }
  sparsity[t] = l1 > 0 ? (double)l1 / sqrt((double)l2sq) : 0.0;
}

}  // namespace

size_t tag_hist_smem_limit() { return (size_t)200 * 1024; }

cudaError_t launch_tag_hist(const int64_t *offsets, const int64_t *tag_off, const int32_t *tags, int K, int V,
                            int64_t *chunk_start, double *colsums, int64_t *counts, double *sparsity, Header *hdr,
                            cudaStream_t s) {
  tag_chunks_kernel<<<1, 1024, 0, s>>>(offsets, tag_off, K, chunk_start, hdr);
  const size_t smem = (size_t)((V + 1) / 2) * sizeof(uint32_t);
  const bool in_smem = smem <= tag_hist_smem_limit();
  const int zb = K < 1024 ? K : 1024;
  tag_zero_kernel<<<zb, 256, 0, s>>>(chunk_start, K, V, !in_smem, counts);
  int grid = num_sms();
  cudaError_t e;
  if (in_smem) {
    e = cudaFuncSetAttribute(tag_hist_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int per_sm = (int)((size_t)(227 * 1024) / (smem + 1024));
    grid *= per_sm < 1 ? 1 : (per_sm > 8 ? 8 : per_sm);
    tag_hist_kernel<true><<<grid, kTagThreads, smem, s>>>(offsets, tag_off, tags, K, V, chunk_start, counts, hdr);
  } else {
    grid *= 4;
    tag_hist_kernel<false><<<grid, kTagThreads, 0, s>>>(offsets, tag_off, tags, K, V, chunk_start, counts, hdr);
  }
  count_launch(3);
  if (sparsity) {
    const int slices = K < kTagSlices ? K : kTagSlices;
    const int rows = (K + slices - 1) / slices;
    const dim3 cg((unsigned)((V + 255) / 256), (unsigned)slices);
    tag_colsum_kernel<<<cg, 256, 0, s>>>(counts, K, V, rows, reinterpret_cast<uint64_t *>(colsums));
    tag_sparsity_kernel<<<(V + 255) / 256, 256, 0, s>>>(reinterpret_cast<const uint64_t *>(colsums), V, slices,
                                                          sparsity);
    count_launch(2);
  }
  return cudaGetLastError();
}

}  // namespace hme
