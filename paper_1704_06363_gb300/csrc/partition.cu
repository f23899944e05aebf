// partition.cu -- each expert's share of the data (Section 2: every expert is
// trained "on its own share of the training data"; Section 2 also says no
// attempt is made to balance the clusters, so buckets can be very unequal).
//
// A stable counting sort of the labels, integer-exact:
//   1. count    each warp owns a contiguous tile of labels and counts it into
//               private shared-memory bins (one shared atomic per label);
//               tile counts go to an ntiles x bins int32 matrix.
//   2. colscan  exclusive prefix of that matrix down each column (per bucket)
//               and the bucket totals.
//   3. offsets  exclusive prefix of the totals.
//   4. scatter  each warp walks its tile again in index order, kChunk labels
//               at a time: every item gets its rank among the chunk's items of
//               its bucket (one ballot per key bit finds the lanes of a round
//               with the same key -- much cheaper than __match_any_sync here),
//               the chunk is reordered by bucket in shared memory, and the
//               items are stored in that order, so consecutive lanes write
//               consecutive slots of a bucket.  An item's slot is offsets[k] +
//               (items of bucket k in earlier tiles and chunks) + its rank, so
//               within a bucket indices ascend.
// With many buckets (K > kOnePassMaxK) a chunk holds too few items per bucket
// for the stores to coalesce, so the sort runs as two stable passes of at
// most 128 buckets, on the low and then the high label bits (a least-
// significant-digit radix sort: the second pass keeps the first one's order
// within a bucket, so the result is ordered by label and, within a label, by
// index); offsets and hist then come from a binary search of the sorted labels.
// Labels are staged kChunk at a time through a per-warp shared buffer with
// 16-byte loads.  Labels outside [0, K) set kStatusBadLabel and are skipped.
#include "hme_common.cuh"

namespace hme {

namespace {

constexpr int kChunk = 512;        // labels staged per warp step

// Per-warp shared layout: [bins, padded to a multiple of 4][kChunk staged labels]
// so that the staging buffer starts on a 16-byte boundary (int4 stores).
__host__ __device__ __forceinline__ int bins_stride(int K) { return (K + 3) / 4 * 4; }
__host__ __device__ __forceinline__ int count_words(int bins) { return bins_stride(bins) + kChunk; }
__host__ __device__ __forceinline__ int scatter_words(int bins) { return 3 * bins_stride(bins) + 4 * kChunk; }
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

// Items of a tile: [start, min(n, start + tile)) with n = min(N, *n_dev) (or
// N).  The bucket of a valid label is (label >> shift) & mask.
__global__ void part_count_kernel(const int32_t *__restrict__ labels, int64_t N, const int64_t *__restrict__ n_dev,
                                  int K, int bins, int shift, int mask, bool check, int64_t tile, int64_t ntiles,
                                  int32_t *__restrict__ tilecnt, Header *hdr, int wpb) {
  extern __shared__ int32_t psm[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t gw = (int64_t)blockIdx.x * wpb + warp;
  if (gw >= ntiles) return;
  int32_t *cnt = psm + (size_t)warp * count_words(bins);
  int32_t *buf = cnt + bins_stride(bins);
  for (int k = lane; k < bins; k += 32) cnt[k] = 0;
  __syncwarp();
  const int64_t n = n_dev ? min(N, *n_dev) : N;
  const int64_t start = gw * tile;
  const int64_t end = min(n, start + tile);
  const bool aligned = (reinterpret_cast<uintptr_t>(labels) & 15u) == 0;
  bool bad = false;
  for (int64_t pos = start; pos < end; pos += kChunk) {
    stage_labels(labels, pos, end, buf, lane, aligned);
    const int rounds = (int)min((int64_t)kChunk, end - pos + 31) / 32;
    for (int r = 0; r < rounds; ++r) {
      const int64_t i = pos + 32 * r + lane;
      const int label = buf[32 * r + lane];
      const bool valid = label >= 0 && label < K;
      if (check && i < end && !valid) bad = true;
      if (i < end && valid) atomicAdd(&cnt[(label >> shift) & mask], 1);
    }
    __syncwarp();
  }
  if (bad) atomicOr(&hdr->status, (uint32_t)kStatusBadLabel);
  for (int k = lane; k < bins; k += 32) tilecnt[gw * bins + k] = cnt[k];
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

// Stable scatter of a tile, kChunk items at a time, reordered by bucket in
// shared memory before the stores: perm_out[slot] = payload ? payload[i] : i,
// labels_out[slot] = label.  Per-warp shared layout: run, cnt, loff (bins
// each, padded), staged labels, staged payload, reordered labels and payload.
__global__ void part_scatter_kernel(const int32_t *__restrict__ labels, const int32_t *__restrict__ payload,
                                    int64_t N, const int64_t *__restrict__ n_dev, int K, int bins, int shift,
                                    int mask, int nbits, int64_t tile, int64_t ntiles,
                                    const int32_t *__restrict__ tileoff, const int64_t *__restrict__ offsets,
                                    int32_t *__restrict__ perm_out, int32_t *__restrict__ labels_out, int wpb) {
  extern __shared__ int32_t psm[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t gw = (int64_t)blockIdx.x * wpb + warp;
  if (gw >= ntiles) return;
  const int bs = bins_stride(bins);
  int32_t *run = psm + (size_t)warp * scatter_words(bins);
  int32_t *cnt = run + bs;
  int32_t *loff = cnt + bs;
  int32_t *buf = loff + bs;
  int32_t *pbuf = buf + kChunk;
  int32_t *olab = pbuf + kChunk;
  int32_t *opay = olab + kChunk;
  for (int k = lane; k < bins; k += 32) run[k] = (int32_t)(offsets[k] + tileoff[gw * bins + k]);
  const int64_t n = n_dev ? min(N, *n_dev) : N;
  const int64_t start = gw * tile;
  const int64_t end = min(n, start + tile);
  const bool aligned = (reinterpret_cast<uintptr_t>(labels) & 15u) == 0;
  const bool paligned = payload && (reinterpret_cast<uintptr_t>(payload) & 15u) == 0;
  const unsigned lt = (1u << lane) - 1u;
  constexpr int R = kChunk / 32;
  for (int64_t pos = start; pos < end; pos += kChunk) {
    for (int k = lane; k < bins; k += 32) cnt[k] = 0;
    stage_labels(labels, pos, end, buf, lane, aligned);
    if (payload) stage_labels(payload, pos, end, pbuf, lane, paligned);
    // rank of every item among the chunk's items of its bucket, in index order
    int key[R], rk[R];
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const int64_t i = pos + 32 * r + lane;
      const int label = buf[32 * r + lane];
      key[r] = (i < end && label >= 0 && label < K) ? (label >> shift) & mask : -1;
      const unsigned peers = same_key_lanes(key[r], nbits);
      rk[r] = key[r] >= 0 ? cnt[key[r]] + __popc(peers & lt) : 0;
      __syncwarp();
      if (key[r] >= 0 && lane == __ffs(peers) - 1) cnt[key[r]] += __popc(peers);
      __syncwarp();
    }
    // loff = exclusive prefix of cnt over the buckets (each lane a run of them)
    const int per = (bins + 31) / 32;
    const int k0 = lane * per, k1 = min(bins, k0 + per);
    int local = 0;
    for (int k = k0; k < k1; ++k) local += cnt[k];
    int incl = local;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += v;
    }
    const int nvalid = __shfl_sync(0xffffffffu, incl, 31);
    int acc = incl - local;
    for (int k = k0; k < k1; ++k) {
      loff[k] = acc;
      acc += cnt[k];
    }
    __syncwarp();
    // reorder the chunk by bucket
#pragma unroll
    for (int r = 0; r < R; ++r) {
      if (key[r] >= 0) {
        const int at = loff[key[r]] + rk[r];
        olab[at] = buf[32 * r + lane];
        opay[at] = payload ? pbuf[32 * r + lane] : (int32_t)(pos + 32 * r + lane);
      }
    }
    __syncwarp();
    // consecutive lanes store consecutive slots of a bucket
    for (int j = lane; j < nvalid; j += 32) {
      const int label = olab[j];
      const int k = (label >> shift) & mask;
      const int32_t slot = run[k] + (j - loff[k]);
      perm_out[slot] = opay[j];
      if (labels_out) labels_out[slot] = label;
    }
    __syncwarp();
    for (int k = lane; k < bins; k += 32) run[k] += cnt[k];
    __syncwarp();
  }
}

// Two-pass partition: offsets[k] = first position of label k in the sorted
// labels (binary search; offsets[K] = items), hist[k] = offsets[k+1] - offsets[k].
__global__ void part_bounds_kernel(const int32_t *__restrict__ sorted, const int64_t *__restrict__ n_dev, int K,
                                   int64_t *__restrict__ hist, int64_t *__restrict__ offsets) {
  const int64_t n = *n_dev;
  auto lower = [&](int k) -> int64_t {
    int64_t lo = 0, hi = n;
    while (lo < hi) {
      const int64_t mid = (lo + hi) >> 1;
      if (__ldg(sorted + mid) < k)
        lo = mid + 1;
      else
        hi = mid;
    }
    return lo;
  };
  for (int k = blockIdx.x * blockDim.x + threadIdx.x; k <= K; k += gridDim.x * blockDim.x) {
    const int64_t a = lower(k);
    offsets[k] = a;
    if (k < K) hist[k] = lower(k + 1) - a;
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

int warps_per_block(int words) {
  const size_t per_warp = (size_t)words * sizeof(int32_t);
  int w = (int)((96 * 1024) / per_warp);
  if (w > 8) w = 8;
  if (w < 1) w = 1;
  return w;
}

}  // namespace

PartLayout part_layout(size_t base, int64_t N, int K) {
  PartLayout pl;
  int nbits = 0;
  while ((1 << nbits) < K) ++nbits;
  pl.two_pass = K > kOnePassMaxK;
  pl.bits1 = pl.two_pass ? (nbits + 1) / 2 : nbits;
  pl.bits2 = pl.two_pass ? nbits - pl.bits1 : 0;
  pl.bins = pl.two_pass ? (1 << pl.bits1) : K;
  int64_t tile = (N + kTargetTiles - 1) / kTargetTiles;
  if (tile < 1024) tile = 1024;
  if (tile < 4 * (int64_t)pl.bins) tile = 4 * (int64_t)pl.bins;
  tile = (tile + kChunk - 1) / kChunk * kChunk;
  pl.tile = tile;
  pl.ntiles = N > 0 ? (N + tile - 1) / tile : 0;
  size_t off = align_up(base, 256);
  pl.tilecnt = off;
  off = align_up(off + (size_t)(pl.ntiles > 0 ? pl.ntiles : 1) * pl.bins * sizeof(int32_t), 256);
  pl.hist = off;
  off = align_up(off + (size_t)K * sizeof(int64_t), 256);
  pl.offs = off;
  off = align_up(off + (size_t)(K + 1) * sizeof(int64_t), 256);
  pl.dig = pl.tmp = 0;
  if (pl.two_pass) {
    pl.dig = off;
    off = align_up(off + (size_t)4 * (pl.bins + 1) * sizeof(int64_t), 256);
    pl.tmp = off;
    off = align_up(off + (size_t)3 * (N > 0 ? N : 1) * sizeof(int32_t), 256);
  }
  pl.misc = off;
  const int64_t nb = (N + kScanItems) / kScanItems + 1;
  off = align_up(off + (size_t)nb * sizeof(int64_t), 256);
  pl.end = off;
  return pl;
}

namespace {

// One stable counting-sort pass over the buckets (label >> shift) & mask.
cudaError_t sort_pass(const int32_t *keys, const int32_t *payload, int64_t N, const int64_t *n_dev, int K, int bins,
                      int shift, int mask, int nbits, bool check, const PartLayout &pl, int32_t *tilecnt,
                      int64_t *hist, int64_t *offsets, int32_t *perm_out, int32_t *labels_out, Header *hdr,
                      cudaStream_t s) {
  const int wc = warps_per_block(count_words(bins)), ws = warps_per_block(scatter_words(bins));
  const size_t smc = (size_t)wc * count_words(bins) * sizeof(int32_t);
  const size_t sms = (size_t)ws * scatter_words(bins) * sizeof(int32_t);
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
    part_count_kernel<<<(unsigned)((pl.ntiles + wc - 1) / wc), 32 * wc, smc, s>>>(
        keys, N, n_dev, K, bins, shift, mask, check, pl.tile, pl.ntiles, tilecnt, hdr, wc);
    count_launch();
  }
  part_colscan_kernel<<<(bins + 31) / 32, 1024, 0, s>>>(tilecnt, pl.ntiles, bins, hist);
  part_offsets_kernel<<<1, 1024, 0, s>>>(hist, bins, offsets);
  count_launch(2);
  if (pl.ntiles > 0) {
    part_scatter_kernel<<<(unsigned)((pl.ntiles + ws - 1) / ws), 32 * ws, sms, s>>>(
        keys, payload, N, n_dev, K, bins, shift, mask, nbits, pl.tile, pl.ntiles, tilecnt, offsets, perm_out,
        labels_out, ws);
    count_launch();
  }
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_partition(const int32_t *labels, int64_t N, int K, const PartLayout &pl, char *ws,
                             int64_t *hist, int64_t *offsets, int32_t *perm, int32_t *sorted_labels, Header *hdr,
                             cudaStream_t s) {
  int32_t *tilecnt = reinterpret_cast<int32_t *>(ws + pl.tilecnt);
  if (!pl.two_pass) {
    int nbits = 0;
    while ((1 << nbits) < K) ++nbits;
    return sort_pass(labels, nullptr, N, nullptr, K, K, 0, 0x7FFFFFFF, nbits, true, pl, tilecnt, hist, offsets,
                     perm, sorted_labels, hdr, s);
  }
  int64_t *dig = reinterpret_cast<int64_t *>(ws + pl.dig);
  int64_t *hist1 = dig, *offs1 = dig + (pl.bins + 1), *hist2 = dig + 2 * (pl.bins + 1),
          *offs2 = dig + 3 * (pl.bins + 1);
  int32_t *tmp = reinterpret_cast<int32_t *>(ws + pl.tmp);
  int32_t *order1 = tmp, *labels1 = tmp + N, *sorted = sorted_labels ? sorted_labels : tmp + 2 * N;
  // pass 1: low bits of the input labels (checked); pass 2: high bits of pass 1's output
  cudaError_t e = sort_pass(labels, nullptr, N, nullptr, K, pl.bins, 0, (1 << pl.bits1) - 1, pl.bits1, true, pl,
                            tilecnt, hist1, offs1, order1, labels1, hdr, s);
  if (e != cudaSuccess) return e;
  const int bins2 = 1 << pl.bits2;
  e = sort_pass(labels1, order1, N, offs1 + pl.bins, K, bins2, pl.bits1, bins2 - 1, pl.bits2, false, pl, tilecnt,
                hist2, offs2, perm, sorted, hdr, s);
  if (e != cudaSuccess) return e;
  part_bounds_kernel<<<(K + 256) / 256, 256, 0, s>>>(sorted, offs1 + pl.bins, K, hist, offsets);
  count_launch();
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
