// partition.cu -- each expert's share of the data (Section 2: every expert is
// trained "on its own share of the training data"; Section 2 also says no
// attempt is made to balance the clusters, so buckets can be very unequal).
//
// A stable counting sort of the labels, integer-exact:
//   1. count    each warp owns a contiguous tile of labels and counts it into
//               private shared-memory bins (one shared atomic per label);
//               tile counts go to an ntiles x K int32 matrix.
//   2. colscan  exclusive prefix of that matrix down each column (per bucket)
//               and the bucket totals hist[k].
//   3. offsets  exclusive prefix of hist -> offsets[0..K].
//   4. scatter  each warp walks its tile again in index order; an item's slot
//               is offsets[k] + (items of bucket k in earlier tiles) + (items
//               of k earlier in this tile), the last part from the running
//               shared-memory bin plus the rank among equal labels of lower
//               lanes in the round.  So within a bucket indices ascend.  The
//               lanes holding the same label are found with one ballot per
//               label bit (ceil(log2 K) ballots), which is much cheaper than
//               __match_any_sync on this hardware.
// Labels are staged 512 at a time through a per-warp shared buffer with
// 16-byte loads.  Labels outside [0, K) set kStatusBadLabel and are skipped.
#include "hme_common.cuh"

namespace hme {

namespace {

constexpr int kChunk = 512;        // labels staged per warp step

// Per-warp shared layout: [bins, padded to a multiple of 4][kChunk staged labels]
// so that the staging buffer starts on a 16-byte boundary (int4 stores).
__host__ __device__ __forceinline__ int bins_stride(int K) { return (K + 3) / 4 * 4; }
__host__ __device__ __forceinline__ int warp_words(int K) { return bins_stride(K) + kChunk; }
constexpr int64_t kTargetTiles = 2432;

__device__ __forceinline__ void stage_labels(const int32_t *__restrict__ labels, int64_t pos, int64_t end,
                                             int32_t *buf, int lane, bool aligned) {
  if (aligned && pos + kChunk <= end) {
    int4 v[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) v[u] = __ldg(reinterpret_cast<const int4 *>(labels + pos + 128 * u + 4 * lane));
#pragma unroll
    for (int u = 0; u < 4; ++u) *reinterpret_cast<int4 *>(buf + 128 * u + 4 * lane) = v[u];
  } else {
    for (int j = lane; j < kChunk; j += 32) buf[j] = (pos + j < end) ? __ldg(labels + pos + j) : -1;
  }
  __syncwarp();
}

// Lanes of the warp whose key equals this lane's key (valid keys are in
// [0, 2^nbits)); keys < 0 match no valid lane and get an empty mask.
__device__ __forceinline__ unsigned same_key_lanes(int key, int nbits) {
  unsigned peers = __ballot_sync(0xffffffffu, key >= 0);
  for (int b = 0; b < nbits; ++b) {
    const bool bit = (key >> b) & 1;
    const unsigned m = __ballot_sync(0xffffffffu, bit);
    peers &= bit ? m : ~m;
  }
  return key >= 0 ? peers : 0u;
}

__global__ void part_count_kernel(const int32_t *__restrict__ labels, int64_t N, int K, int64_t tile,
                                  int64_t ntiles, int32_t *__restrict__ tilecnt, Header *hdr, int wpb) {
  extern __shared__ int32_t psm[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t gw = (int64_t)blockIdx.x * wpb + warp;
  if (gw >= ntiles) return;
  int32_t *bins = psm + (size_t)warp * warp_words(K);
  int32_t *buf = bins + bins_stride(K);
  for (int k = lane; k < K; k += 32) bins[k] = 0;
  __syncwarp();
  const int64_t start = gw * tile;
  const int64_t end = min(N, start + tile);
  const bool aligned = (reinterpret_cast<uintptr_t>(labels) & 15u) == 0;
  bool bad = false;
  for (int64_t pos = start; pos < end; pos += kChunk) {
    stage_labels(labels, pos, end, buf, lane, aligned);
    const int rounds = (int)min((int64_t)kChunk, end - pos + 31) / 32;
    for (int r = 0; r < rounds; ++r) {
      const int64_t i = pos + 32 * r + lane;
      const int key = buf[32 * r + lane];
      if (i < end && (key < 0 || key >= K)) bad = true;
      if (i < end && key >= 0 && key < K) atomicAdd(&bins[key], 1);
    }
    __syncwarp();
  }
  if (bad) atomicOr(&hdr->status, (uint32_t)kStatusBadLabel);
  for (int k = lane; k < K; k += 32) tilecnt[gw * K + k] = bins[k];
}

// Exclusive prefix down each column of the ntiles x K matrix; hist[k] = column total.
__global__ void __launch_bounds__(1024) part_colscan_kernel(int32_t *__restrict__ m, int64_t ntiles, int K,
                                                            int64_t *__restrict__ hist) {
  __shared__ int64_t part[32][33];
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  const int col = blockIdx.x * 32 + tx;
  const int64_t R = (ntiles + 31) / 32;
  const int64_t r0 = ty * R, r1 = min(ntiles, r0 + R);
  int64_t sum = 0;
  if (col < K)
    for (int64_t r = r0; r < r1; ++r) sum += m[r * K + col];
  part[ty][tx] = sum;
  __syncthreads();
  if (ty == 0) {
    int64_t run = 0;
    for (int g = 0; g < 32; ++g) {
      const int64_t v = part[g][tx];
      part[g][tx] = run;
      run += v;
    }
    if (col < K) hist[col] = run;
  }
  __syncthreads();
  if (col < K) {
    int64_t run = part[ty][tx];
    for (int64_t r = r0; r < r1; ++r) {
      const int32_t v = m[r * K + col];
      m[r * K + col] = (int32_t)run;
      run += v;
    }
  }
}

// offsets[0..K] = exclusive prefix of hist (one block).
__global__ void __launch_bounds__(1024) part_offsets_kernel(const int64_t *__restrict__ hist, int K,
                                                            int64_t *__restrict__ offsets) {
  __shared__ int64_t wsum[32];
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const int per = (K + 1023) / 1024;
  const int k0 = t * per, k1 = min(K, k0 + per);
  int64_t local = 0;
  for (int k = k0; k < k1; ++k) local += hist[k];
  int64_t incl = local;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int64_t v = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += v;
  }
  if (lane == 31) wsum[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    int64_t w = wsum[lane];
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
    offsets[k] = run;
    run += hist[k];
  }
  if (t == 1023) offsets[K] = run;
}

__global__ void part_scatter_kernel(const int32_t *__restrict__ labels, int64_t N, int K, int nbits, int64_t tile,
                                    int64_t ntiles, const int32_t *__restrict__ tileoff,
                                    const int64_t *__restrict__ offsets, int32_t *__restrict__ perm,
                                    int32_t *__restrict__ sorted_labels, int wpb) {
  extern __shared__ int32_t psm[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t gw = (int64_t)blockIdx.x * wpb + warp;
  if (gw >= ntiles) return;
  int32_t *run = psm + (size_t)warp * warp_words(K);
  int32_t *buf = run + bins_stride(K);
  for (int k = lane; k < K; k += 32) run[k] = (int32_t)(offsets[k] + tileoff[gw * K + k]);
  __syncwarp();
  const int64_t start = gw * tile;
  const int64_t end = min(N, start + tile);
  const bool aligned = (reinterpret_cast<uintptr_t>(labels) & 15u) == 0;
  const unsigned lt = (1u << lane) - 1u;
  for (int64_t pos = start; pos < end; pos += kChunk) {
    stage_labels(labels, pos, end, buf, lane, aligned);
    const int rounds = (int)min((int64_t)kChunk, end - pos + 31) / 32;
    for (int r = 0; r < rounds; ++r) {
      const int64_t i = pos + 32 * r + lane;
      int key = buf[32 * r + lane];
      if (i >= end || key < 0 || key >= K) key = -1;
      const unsigned peers = same_key_lanes(key, nbits);
      if (key >= 0) {
        const int32_t slot = run[key] + __popc(peers & lt);
        perm[slot] = (int32_t)i;
        if (sorted_labels) sorted_labels[slot] = key;
      }
      __syncwarp();
      if (key >= 0 && lane == __ffs(peers) - 1) run[key] += __popc(peers);
      __syncwarp();
    }
    __syncwarp();
  }
}

// ---- moving the CSR tag lists with their points --------------------------

__global__ void tag_len_kernel(const int32_t *__restrict__ perm, int64_t N, const int64_t *__restrict__ valid_total,
                               const int64_t *__restrict__ tag_off, int64_t *__restrict__ out) {
  const int64_t s = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (s == 0) out[0] = 0;
  if (s < N) {
    int64_t len = 0;
    if (s < *valid_total) {
      const int64_t p = perm[s];
      len = tag_off[p + 1] - tag_off[p];
    }
    out[s + 1] = len;
  }
}

constexpr int kScanItems = 2048;  // per block, 1024 threads x 2

__device__ __forceinline__ int64_t block_incl_scan(int64_t v, int64_t *wsum) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int64_t u = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += u;
  }
  if (lane == 31) wsum[warp] = v;
  __syncthreads();
  if (warp == 0) {
    int64_t w = wsum[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int64_t u = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += u;
    }
    wsum[lane] = w;
  }
  __syncthreads();
  const int64_t add = warp > 0 ? wsum[warp - 1] : 0;
  __syncthreads();
  return v + add;
}

// Block sums of a[0..n).
__global__ void __launch_bounds__(1024) scan_blocksum_kernel(const int64_t *__restrict__ a, int64_t n,
                                                             int64_t *__restrict__ bs) {
  __shared__ int64_t wsum[32];
  const int64_t i0 = (int64_t)blockIdx.x * kScanItems + 2 * threadIdx.x;
  int64_t v = 0;
  if (i0 < n) v += a[i0];
  if (i0 + 1 < n) v += a[i0 + 1];
  const int64_t tot = block_incl_scan(v, wsum);
  if (threadIdx.x == 1023) bs[blockIdx.x] = tot;
}

// Exclusive scan of the block sums in place (one block).
__global__ void __launch_bounds__(1024) scan_top_kernel(int64_t *__restrict__ bs, int64_t nb) {
  __shared__ int64_t wsum[32];
  __shared__ int64_t carry;
  if (threadIdx.x == 0) carry = 0;
  __syncthreads();
  for (int64_t b0 = 0; b0 < nb; b0 += 1024) {
    const int64_t i = b0 + threadIdx.x;
    const int64_t v = i < nb ? bs[i] : 0;
    const int64_t incl = block_incl_scan(v, wsum);
    const int64_t c = carry;
    if (i < nb) bs[i] = c + incl - v;
    __syncthreads();
    if (threadIdx.x == 1023) carry = c + incl;
    __syncthreads();
  }
}

// Inclusive scan of a[0..n) in place, block offsets from bs.
__global__ void __launch_bounds__(1024) scan_apply_kernel(int64_t *__restrict__ a, int64_t n,
                                                          const int64_t *__restrict__ bs) {
  __shared__ int64_t wsum[32];
  const int64_t i0 = (int64_t)blockIdx.x * kScanItems + 2 * threadIdx.x;
  const int64_t v0 = i0 < n ? a[i0] : 0;
  const int64_t v1 = i0 + 1 < n ? a[i0 + 1] : 0;
  const int64_t incl = block_incl_scan(v0 + v1, wsum);
  const int64_t base = bs[blockIdx.x] + incl - v0 - v1;
  if (i0 < n) a[i0] = base + v0;
  if (i0 + 1 < n) a[i0 + 1] = base + v0 + v1;
}

__global__ void tag_copy_kernel(const int32_t *__restrict__ perm, int64_t N,
                                const int64_t *__restrict__ valid_total, const int64_t *__restrict__ tag_off,
                                const int32_t *__restrict__ tags, const int64_t *__restrict__ tag_off_out,
                                int32_t *__restrict__ tags_out) {
  const int64_t s = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (s >= N || s >= *valid_total) return;
  const int64_t p = perm[s];
  const int64_t src = tag_off[p], len = tag_off[p + 1] - src, dst = tag_off_out[s];
  for (int64_t t = 0; t < len; ++t) tags_out[dst + t] = tags[src + t];
}

int warps_per_block(int K) {
  const size_t per_warp = (size_t)warp_words(K) * sizeof(int32_t);
  int w = (int)((96 * 1024) / per_warp);
  if (w > 8) w = 8;
  if (w < 1) w = 1;
  return w;
}

}  // namespace

PartLayout part_layout(size_t base, int64_t N, int K) {
  PartLayout pl;
  int64_t tile = (N + kTargetTiles - 1) / kTargetTiles;
  if (tile < 1024) tile = 1024;
  if (tile < 4 * (int64_t)K) tile = 4 * (int64_t)K;
  tile = (tile + kChunk - 1) / kChunk * kChunk;
  pl.tile = tile;
  pl.ntiles = N > 0 ? (N + tile - 1) / tile : 0;
  size_t off = align_up(base, 256);
  pl.tilecnt = off;
  off = align_up(off + (size_t)(pl.ntiles > 0 ? pl.ntiles : 1) * K * sizeof(int32_t), 256);
  pl.hist = off;
  off = align_up(off + (size_t)K * sizeof(int64_t), 256);
  pl.offs = off;
  off = align_up(off + (size_t)(K + 1) * sizeof(int64_t), 256);
  pl.misc = off;
  const int64_t nb = (N + kScanItems) / kScanItems + 1;
  off = align_up(off + (size_t)nb * sizeof(int64_t), 256);
  pl.end = off;
  return pl;
}

cudaError_t launch_partition(const int32_t *labels, int64_t N, int K, const PartLayout &pl, char *ws,
                             int64_t *hist, int64_t *offsets, int32_t *perm, int32_t *sorted_labels, Header *hdr,
                             cudaStream_t s) {
  int32_t *tilecnt = reinterpret_cast<int32_t *>(ws + pl.tilecnt);
  const int wpb = warps_per_block(K);
  const size_t smem = (size_t)wpb * warp_words(K) * sizeof(int32_t);
  cudaError_t e;
  if (smem > 48 * 1024) {
    e = cudaFuncSetAttribute(part_count_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(part_scatter_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  const unsigned blocks = (unsigned)((pl.ntiles + wpb - 1) / wpb);
  if (pl.ntiles > 0) {
    part_count_kernel<<<blocks, 32 * wpb, smem, s>>>(labels, N, K, pl.tile, pl.ntiles, tilecnt, hdr, wpb);
    count_launch();
  }
  part_colscan_kernel<<<(K + 31) / 32, 1024, 0, s>>>(tilecnt, pl.ntiles, K, hist);
  part_offsets_kernel<<<1, 1024, 0, s>>>(hist, K, offsets);
  count_launch(2);
  if (pl.ntiles > 0) {
    int nbits = 0;
    while ((1 << nbits) < K) ++nbits;
    part_scatter_kernel<<<blocks, 32 * wpb, smem, s>>>(labels, N, K, nbits, pl.tile, pl.ntiles, tilecnt, offsets,
                                                       perm, sorted_labels, wpb);
    count_launch();
  }
  return cudaGetLastError();
}

cudaError_t launch_tag_scatter(const int32_t *perm, int64_t N, const int64_t *valid_total, const int64_t *tag_off,
                               const int32_t *tags, int64_t *tag_off_out, int32_t *tags_out, int64_t *scratch,
                               int64_t nscratch, cudaStream_t s) {
  const unsigned g = (unsigned)((N + 255) / 256 + (N == 0 ? 1 : 0));
  tag_len_kernel<<<g, 256, 0, s>>>(perm, N, valid_total, tag_off, tag_off_out);
  count_launch();
  if (N > 0) {
    const int64_t nb = (N + kScanItems - 1) / kScanItems;
    if (nb > nscratch) return cudaErrorInvalidValue;
    scan_blocksum_kernel<<<(unsigned)nb, 1024, 0, s>>>(tag_off_out + 1, N, scratch);
    scan_top_kernel<<<1, 1024, 0, s>>>(scratch, nb);
    scan_apply_kernel<<<(unsigned)nb, 1024, 0, s>>>(tag_off_out + 1, N, scratch);
    tag_copy_kernel<<<g, 256, 0, s>>>(perm, N, valid_total, tag_off, tags, tag_off_out, tags_out);
    count_launch(4);
  }
  return cudaGetLastError();
}

}  // namespace hme
