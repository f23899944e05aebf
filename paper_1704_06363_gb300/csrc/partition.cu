// partition.cu -- each expert's share of the data (Section 2: every expert is
// trained "on its own share of the training data"; Section 2 also says no
// attempt is made to balance the clusters, so buckets can be very unequal).
//
// A stable counting sort of the labels, integer-exact, in one pass over the
// items for every K (up to 16384):
//   1. count    the items are cut into ntiles contiguous tiles, one CTA each
//               (two per SM); a CTA counts its tile into a shared-memory
//               histogram of K bins and writes its row of the ntiles x K
//               matrix of tile counts.
//   2. colscan  exclusive prefix of that matrix down each column (per bucket)
//               and the bucket totals (hist).
//   3. offsets  exclusive prefix of hist.
//   4. scatter  each CTA walks its tile in index order, kPChunk items at a
//               time.  A chunk is sorted by label inside shared memory with a
//               stable least-significant-digit radix sort of one or two
//               passes (digits of at most 8 bits; each warp ranks its items
//               with one ballot per digit bit, then one block-wide scan over
//               (digit, warp) gives every item its place), so that items of a
//               bucket become one run, in index order.  The CTA keeps one
//               output cursor per bucket, offsets[k] + (items of bucket k in
//               earlier tiles) + (items already placed by this tile); the run
//               of bucket k is stored at cursor[k], cursor[k] + 1, ... by
//               consecutive threads, so stores coalesce wherever a bucket has
//               several items in a chunk, and each tile advances one write
//               front per bucket: ntiles x K fronts, few enough for L2 to
//               gather the partial sectors before they go to DRAM.
// Within a bucket indices ascend (the tile order, then the chunk order, then
// the stable sort), which is the definition of the stable partition.  Labels
// outside [0, K) set kStatusBadLabel in the count pass and are sorted behind
// every valid label by the scatter, which stores none of them.
#include "hme_common.cuh"

namespace hme {

namespace {

constexpr int kPThreads = 512;                // threads of a count / scatter CTA
constexpr int kPWarps = kPThreads / 32;
constexpr int kPR = kPartChunk / kPThreads;   // items per thread per chunk
constexpr int kMaxDigitBits = 8;
constexpr int kPartTilesPerSM = 2;
constexpr int kPartSMs = 152;                 // GB300: the tile count fills two CTAs per SM
static_assert(kPartChunk % kPThreads == 0 && kPartChunk <= 65536, "chunk positions fit 16 bits");

__host__ __device__ __forceinline__ int round4(int k) { return (k + 3) / 4 * 4; }

// Shared-memory words of the scatter CTA: cursors, two key buffers, the
// per-warp digit counts (rows of 2^bmax + 1 words: the scan walks them
// column-wise without bank conflicts) and the scan's warp totals.
__host__ __device__ __forceinline__ size_t scatter_smem_words(int K, int bmax) {
  return (size_t)round4(K) + 2 * (size_t)kPartChunk + (size_t)kPWarps * ((1 << bmax) + 1) + 32;
}

// Count each tile into a shared-memory histogram and write its row of tile counts.
__global__ void __launch_bounds__(kPThreads) part_count_kernel(const int32_t *__restrict__ labels, int64_t N, int K,
                                                               int64_t tile, int32_t *__restrict__ tilecnt,
                                                               Header *hdr) {
  extern __shared__ int32_t hcnt[];
  for (int k = threadIdx.x; k < K; k += kPThreads) hcnt[k] = 0;
  __syncthreads();
  const int64_t start = (int64_t)blockIdx.x * tile;
  const int64_t end = min(N, start + tile);
  bool bad = false;
  auto take = [&](int v) {
    if (v >= 0 && v < K)
      atomicAdd(&hcnt[v], 1);
    else
      bad = true;
  };
  // start is a multiple of kPartChunk, so an aligned base keeps every int4 aligned
  if ((reinterpret_cast<uintptr_t>(labels) & 15u) == 0) {
    const int64_t nvec = (end - start) / 4;
    const int4 *v4 = reinterpret_cast<const int4 *>(labels + start);
    int64_t j = threadIdx.x;
    for (; j + 3 * kPThreads < nvec; j += 4 * kPThreads) {
      int4 v[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) v[u] = __ldg(v4 + j + u * kPThreads);
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        take(v[u].x);
        take(v[u].y);
        take(v[u].z);
        take(v[u].w);
      }
    }
    for (; j < nvec; j += kPThreads) {
      const int4 v = __ldg(v4 + j);
      take(v.x);
      take(v.y);
      take(v.z);
      take(v.w);
    }
    for (int64_t i = start + 4 * nvec + threadIdx.x; i < end; i += kPThreads) take(__ldg(labels + i));
  } else {
    for (int64_t i = start + threadIdx.x; i < end; i += kPThreads) take(__ldg(labels + i));
  }
  if (bad) atomicOr(&hdr->status, (uint32_t)kStatusBadLabel);
  __syncthreads();
  int32_t *row = tilecnt + (int64_t)blockIdx.x * K;
  for (int k = threadIdx.x; k < K; k += kPThreads) row[k] = hcnt[k];
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

// Lanes of the warp whose digit equals this lane's (digits in [0, 2^b)).
__device__ __forceinline__ unsigned same_digit_lanes(unsigned dig, int b) {
  unsigned peers = 0xffffffffu;
  for (int i = 0; i < b; ++i) {
    const unsigned bit = (dig >> i) & 1u;
    const unsigned m = __ballot_sync(0xffffffffu, bit);
    peers &= bit ? m : ~m;
  }
  return peers;
}

// One stable counting pass of the block-local radix sort.  Item r of this
// thread sits at position warp * 32 kPR + 32 r + lane of the current order
// and has packed value v[r] = key << 16 | (position in the chunk's index
// order); its digit is (key >> shift) mod 2^b.  Every item is written to
// out[its position in the order by (digit, current position)].
__device__ __forceinline__ void rank_pass(const uint32_t (&v)[kPR], uint32_t *out, int shift, int b, int32_t *wcnt,
                                          int32_t *wsum) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nd = 1 << b, stride = nd + 1;
  int32_t *mine = wcnt + warp * stride;
  for (int g = lane; g < nd; g += 32) mine[g] = 0;
  __syncwarp();
  const unsigned lt = (1u << lane) - 1u;
  unsigned dig[kPR];
  int rk[kPR];
#pragma unroll
  for (int r = 0; r < kPR; ++r) {
    dig[r] = (v[r] >> (16 + shift)) & (unsigned)(nd - 1);
    const unsigned peers = same_digit_lanes(dig[r], b);
    const int before = mine[dig[r]];
    rk[r] = before + __popc(peers & lt);
    __syncwarp();
    if (lane == __ffs(peers) - 1) mine[dig[r]] = before + __popc(peers);
    __syncwarp();
  }
  __syncthreads();
  // exclusive scan over the (digit, warp) counts, digit-major
  const int n = nd * kPWarps;
  const int per = (n + kPThreads - 1) / kPThreads;
  const int e0 = threadIdx.x * per, e1 = min(n, e0 + per);
  int local = 0;
  for (int e = e0; e < e1; ++e) local += wcnt[(e % kPWarps) * stride + e / kPWarps];
  int incl = local;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int t = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += t;
  }
  if (lane == 31) wsum[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    const int w = lane < kPWarps ? wsum[lane] : 0;
    int wi = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int t = __shfl_up_sync(0xffffffffu, wi, o);
      if (lane >= o) wi += t;
    }
    if (lane < kPWarps) wsum[lane] = wi - w;
  }
  __syncthreads();
  int run = wsum[warp] + incl - local;
  for (int e = e0; e < e1; ++e) {
    int32_t *c = wcnt + (e % kPWarps) * stride + e / kPWarps;
    const int t = *c;
    *c = run;
    run += t;
  }
  __syncthreads();
#pragma unroll
  for (int r = 0; r < kPR; ++r) out[mine[dig[r]] + rk[r]] = v[r];
  __syncthreads();
}

// The stable scatter (see the file comment).  perm_out[slot] = item index,
// labels_out[slot] = label (may be NULL).
__global__ void __launch_bounds__(kPThreads, kPartTilesPerSM) part_scatter_kernel(const int32_t *__restrict__ labels, int64_t N, int K,
                                                                 int b0, int b1, int64_t tile,
                                                                 const int32_t *__restrict__ tileoff,
                                                                 const int64_t *__restrict__ offsets,
                                                                 int32_t *__restrict__ perm_out,
                                                                 int32_t *__restrict__ labels_out) {
  extern __shared__ uint32_t psm[];
  int32_t *cursor = reinterpret_cast<int32_t *>(psm);
  uint32_t *ka = psm + round4(K);
  uint32_t *kb = ka + kPartChunk;
  int32_t *wcnt = reinterpret_cast<int32_t *>(kb + kPartChunk);
  const int bmax = b0 > b1 ? b0 : b1;
  int32_t *wsum = wcnt + kPWarps * ((1 << bmax) + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t t = blockIdx.x;
  for (int k = threadIdx.x; k < K; k += kPThreads) cursor[k] = (int32_t)(offsets[k] + tileoff[t * K + k]);
  const int64_t start = t * tile;
  const int64_t end = min(N, start + tile);
  // item r of a thread: chunk position warp * 32 kPR + 32 r + lane (32 consecutive labels per warp load)
  const int pbase = warp * 32 * kPR + lane;
  int32_t lab[kPR];
#pragma unroll
  for (int r = 0; r < kPR; ++r) {
    const int64_t i = start + pbase + 32 * r;
    lab[r] = i < end ? __ldg(labels + i) : -1;
  }
  for (int64_t pos = start; pos < end; pos += kPartChunk) {
    uint32_t v[kPR];
#pragma unroll
    for (int r = 0; r < kPR; ++r) {
      const unsigned key = (lab[r] >= 0 && lab[r] < K) ? (unsigned)lab[r] : (unsigned)K;
      v[r] = (key << 16) | (unsigned)(pbase + 32 * r);
    }
    // the next chunk's labels are in flight during the sort of this one
    const int64_t nxt = pos + kPartChunk;
#pragma unroll
    for (int r = 0; r < kPR; ++r) {
      const int64_t i = nxt + pbase + 32 * r;
      lab[r] = i < end ? __ldg(labels + i) : -1;
    }
    rank_pass(v, kb, 0, b0, wcnt, wsum);
    const uint32_t *sorted = kb;
    if (b1 > 0) {
      uint32_t w[kPR];
#pragma unroll
      for (int r = 0; r < kPR; ++r) w[r] = kb[pbase + 32 * r];
      rank_pass(w, ka, b0, b1, wcnt, wsum);
      sorted = ka;
    }
    // runs of equal keys: the first item of a run turns the bucket's cursor
    // into its base (cursor - position), every item stores at base + position,
    // the last item moves the cursor past the run
    uint32_t sv[kPR];
    bool last[kPR];
#pragma unroll
    for (int j = 0; j < kPR; ++j) {
      const int q = threadIdx.x + kPThreads * j;
      sv[j] = sorted[q];
      const unsigned key = sv[j] >> 16;
      const unsigned prev = q > 0 ? (sorted[q - 1] >> 16) : 0xFFFFFFFFu;
      const unsigned next = q + 1 < kPartChunk ? (sorted[q + 1] >> 16) : 0xFFFFFFFFu;
      last[j] = key != next;
      if (key < (unsigned)K && key != prev) cursor[key] -= q;
    }
    __syncthreads();
    int32_t slot[kPR];
#pragma unroll
    for (int j = 0; j < kPR; ++j) {
      const int q = threadIdx.x + kPThreads * j;
      const unsigned key = sv[j] >> 16;
      slot[j] = -1;
      if (key < (unsigned)K) {
        slot[j] = cursor[key] + q;
        perm_out[slot[j]] = (int32_t)(pos + (sv[j] & 0xFFFFu));
        if (labels_out) labels_out[slot[j]] = (int32_t)key;
      }
    }
    __syncthreads();
#pragma unroll
    for (int j = 0; j < kPR; ++j)
      if (slot[j] >= 0 && last[j]) cursor[sv[j] >> 16] = slot[j] + 1;
    // the next chunk's first rank pass synchronises before its key buffer is read here again
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

}  // namespace

PartLayout part_layout(size_t base, int64_t N, int K) {
  PartLayout pl;
  int bits = 0;
  while ((1 << bits) < K + 1) ++bits;  // labels 0 .. K-1 and the key K of an invalid label
  pl.b0 = bits <= kMaxDigitBits ? bits : bits / 2;
  pl.b1 = bits - pl.b0;
  int64_t tile = (N + kPartTilesPerSM * kPartSMs - 1) / (kPartTilesPerSM * kPartSMs);
  tile = (tile + kPartChunk - 1) / kPartChunk * kPartChunk;
  if (tile < kPartChunk) tile = kPartChunk;
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
  const size_t smc = (size_t)K * sizeof(int32_t);
  const int bmax = pl.b0 > pl.b1 ? pl.b0 : pl.b1;
  const size_t sms = scatter_smem_words(K, bmax) * sizeof(uint32_t);
  cudaError_t e;
  if (smc > 48 * 1024) {
    e = cudaFuncSetAttribute(part_count_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smc);
    if (e != cudaSuccess) return e;
  }
  if (sms > 48 * 1024) {
    e = cudaFuncSetAttribute(part_scatter_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sms);
    if (e != cudaSuccess) return e;
  }
  if (pl.ntiles > 0) {
    part_count_kernel<<<(unsigned)pl.ntiles, kPThreads, smc, s>>>(labels, N, K, pl.tile, tilecnt, hdr);
    count_launch();
  }
  part_colscan_kernel<<<(K + 31) / 32, 1024, 0, s>>>(tilecnt, pl.ntiles, K, hist);
  part_offsets_kernel<<<1, 1024, 0, s>>>(hist, K, offsets);
  count_launch(2);
  if (pl.ntiles > 0) {
    part_scatter_kernel<<<(unsigned)pl.ntiles, kPThreads, sms, s>>>(labels, N, K, pl.b0, pl.b1, pl.tile, tilecnt,
                                                                    offsets, perm, sorted_labels);
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
