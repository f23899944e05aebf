// partition.cu -- each expert's share of the data (Section 2: every expert is
// trained "on its own share of the training data"; Section 2 also says no
// attempt is made to balance the clusters, so buckets can be very unequal).
//
// A stable counting sort of the labels, integer-exact, in one pass over the
// items for every K (up to 16384):
//   1. count    the items are cut into ntiles contiguous tiles, one CTA each
//               (two per SM, or one when tag lists move along); a CTA
//               counts its tile into a shared-memory
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
//   5. labels   the sorted labels, when asked for, are a fill of each
//               bucket's slot range [offsets[k], offsets[k+1]) with k:
//               sequential 16-byte stores instead of a second scatter.
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
constexpr size_t kMaxSmemScatter = 227 * 1024;
static_assert(kPartChunk % kPThreads == 0 && kPartChunk <= 65536, "chunk positions fit 16 bits");

__host__ __device__ __forceinline__ int round4(int k) { return (k + 3) / 4 * 4; }

// Shared-memory layout of the scatter CTA, in 32-bit words: cursors, two key
// buffers, the per-warp digit counts (rows of 2^bmax + 1 words: the scan
// walks them column-wise without bank conflicts), the scan's warp totals and
// (tag lists) the 16 kPR segment sums of the tag-length scan (int64, at an
// even word).
__host__ __device__ __forceinline__ size_t scatter_wsum_word(int K, int bmax) {
  return (size_t)round4(K) + 2 * (size_t)kPartChunk + (size_t)kPWarps * ((1 << bmax) + 1);
}
__host__ __device__ __forceinline__ size_t scatter_segsum_word(int K, int bmax) {
  return (scatter_wsum_word(K, bmax) + 32 + 1) & ~(size_t)1;
}
// tag lists: the chunk's staged offsets int64[kPartChunk + 1], the list
// destinations by item int64[kPartChunk], and (when it fits) the tag cursors
// int64[K], from an even word
__host__ __device__ __forceinline__ size_t scatter_toff_word(int K, int bmax) {
  return scatter_segsum_word(K, bmax) + 2 * (size_t)kPR * kPWarps;
}
__host__ __device__ __forceinline__ size_t scatter_smem_words(int K, int bmax, bool tags = false,
                                                             bool tcur_smem = false) {
  if (!tags) return scatter_toff_word(K, bmax);
  return scatter_toff_word(K, bmax) + 2 * (size_t)(kPartChunk + 2) + 2 * (size_t)kPartChunk +
         (tcur_smem ? 2 * (size_t)K : 0);
}

// Count each tile into a shared-memory histogram and write its row of tile
// counts; with TAGS also the tile's tag-list lengths per bucket.
template <bool TAGS>
__global__ void __launch_bounds__(kPThreads) part_count_kernel(const int32_t *__restrict__ labels, int64_t N, int K,
                                                               int64_t tile, int32_t *__restrict__ tilecnt,
                                                               const int64_t *__restrict__ tag_off,
                                                               int64_t *__restrict__ tagcnt, Header *hdr) {
  extern __shared__ int32_t hcnt[];
  // tag-list lengths per bucket: 32-bit counters when the tile's lists hold
  // fewer than 2^32 tags in all (64-bit shared atomics are much slower)
  unsigned long long *tcnt = reinterpret_cast<unsigned long long *>(hcnt + round4(K));
  unsigned *tcnt32 = reinterpret_cast<unsigned *>(tcnt);
  const int64_t start = (int64_t)blockIdx.x * tile;
  const int64_t end = min(N, start + tile);
  const bool narrow = !TAGS || (__ldg(tag_off + end) - __ldg(tag_off + start)) < ((int64_t)1 << 32);
  for (int k = threadIdx.x; k < K; k += kPThreads) {
    hcnt[k] = 0;
    if (TAGS) tcnt[k] = 0;
  }
  __syncthreads();
  bool bad = false;
  auto take = [&](int v, int64_t i) {
    if (v >= 0 && v < K) {
      atomicAdd(&hcnt[v], 1);
      if (TAGS) {
        const int64_t len = __ldg(tag_off + i + 1) - __ldg(tag_off + i);
        if (narrow)
          atomicAdd(&tcnt32[v], (unsigned)len);
        else
          atomicAdd(&tcnt[v], (unsigned long long)len);
      }
    } else {
      bad = true;
    }
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
        const int64_t i = start + 4 * (j + u * kPThreads);
        take(v[u].x, i);
        take(v[u].y, i + 1);
        take(v[u].z, i + 2);
        take(v[u].w, i + 3);
      }
    }
    for (; j < nvec; j += kPThreads) {
      const int4 v = __ldg(v4 + j);
      const int64_t i = start + 4 * j;
      take(v.x, i);
      take(v.y, i + 1);
      take(v.z, i + 2);
      take(v.w, i + 3);
    }
    for (int64_t i = start + 4 * nvec + threadIdx.x; i < end; i += kPThreads) take(__ldg(labels + i), i);
  } else {
    for (int64_t i = start + threadIdx.x; i < end; i += kPThreads) take(__ldg(labels + i), i);
  }
  if (bad) atomicOr(&hdr->status, (uint32_t)kStatusBadLabel);
  __syncthreads();
  int32_t *row = tilecnt + (int64_t)blockIdx.x * K;
  for (int k = threadIdx.x; k < K; k += kPThreads) {
    row[k] = hcnt[k];
    if (TAGS) tagcnt[(int64_t)blockIdx.x * K + k] = narrow ? (int64_t)tcnt32[k] : (int64_t)tcnt[k];
  }
}

// Exclusive prefix down each column of the ntiles x K matrix; hist[k] = column total.
template <typename T>
__global__ void __launch_bounds__(1024) part_colscan_kernel(T *__restrict__ m, int64_t ntiles, int K,
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
      const T v = m[r * K + col];
      m[r * K + col] = (T)run;
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

// Lanes of the warp whose digit equals this lane's (digits in [0, 2^B)).
template <int B>
__device__ __forceinline__ unsigned same_digit_lanes(unsigned dig) {
  unsigned peers = 0xffffffffu;
#pragma unroll
  for (int i = 0; i < B; ++i) {
    const bool bit = (dig >> i) & 1u;
    const unsigned m = __ballot_sync(0xffffffffu, bit);
    peers &= bit ? m : ~m;
  }
  return peers;
}

// One stable counting pass of the block-local radix sort.  Item r of this
// thread sits at position warp * 32 kPR + 32 r + lane of the current order
// and has packed value v[r] = key << 16 | (position in the chunk's index
// order); its digit is (key >> SHIFT) mod 2^B.  Every item is written to
// out[its position in the order by (digit, current position)].
template <int B, int SHIFT>
__device__ __forceinline__ void rank_pass(const uint32_t (&v)[kPR], uint32_t *out, int32_t *wcnt, int32_t *wsum) {
  constexpr int ND = 1 << B, STRIDE = ND + 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int32_t *mine = wcnt + warp * STRIDE;
#pragma unroll
  for (int g = lane; g < ND; g += 32) mine[g] = 0;
  __syncwarp();
  const unsigned lt = (1u << lane) - 1u;
  unsigned dig[kPR];
  int rk[kPR];
#pragma unroll
  for (int r = 0; r < kPR; ++r) {
    dig[r] = (v[r] >> (16 + SHIFT)) & (unsigned)(ND - 1);
    const unsigned peers = same_digit_lanes<B>(dig[r]);
    const int before = mine[dig[r]];
    rk[r] = before + __popc(peers & lt);
    __syncwarp();
    if ((peers & lt) == 0) mine[dig[r]] = before + __popc(peers);  // the lowest lane of the group
    __syncwarp();
  }
  __syncthreads();
  // exclusive scan over the (digit, warp) counts, digit-major: entry e is
  // (digit e / kPWarps, warp e % kPWarps)
  constexpr int NE = ND * kPWarps;
  constexpr int PER = (NE + kPThreads - 1) / kPThreads;
  const int e0 = threadIdx.x * PER;
  int cv[PER];
  int local = 0;
#pragma unroll
  for (int u = 0; u < PER; ++u) {
    const int e = e0 + u;
    cv[u] = e < NE ? wcnt[(e % kPWarps) * STRIDE + e / kPWarps] : 0;
    local += cv[u];
  }
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
#pragma unroll
  for (int u = 0; u < PER; ++u) {
    const int e = e0 + u;
    if (e < NE) wcnt[(e % kPWarps) * STRIDE + e / kPWarps] = run;
    run += cv[u];
  }
  __syncthreads();
#pragma unroll
  for (int r = 0; r < kPR; ++r) out[mine[dig[r]] + rk[r]] = v[r];
  __syncthreads();
}

// Tag lists move with their points (TAGS).  The chunk's tag offsets are
// staged in shared memory (cp.async, under the sort).  The list lengths, in
// sorted order, get a block-wide exclusive prefix P; a bucket's tag cursor
// (tag_base[k] + tags of bucket k in earlier tiles + tags this tile has
// placed; in shared memory when K allows, else in the CTA's row of the scanned
// tag-count matrix, which only this CTA touches) advances run by run exactly
// like the item cursor, so the lists of a run land back to back:
// tag_off_out[slot] = the destination of the point's list.  The tags are then
// copied in source order: each warp walks its items 32 at a time, whose
// lists are one contiguous source range (minus those of invalid labels);
// lane l copies tags l, l + 32, ... of it, finding the owning item by a
// binary search over the 32 list starts (shuffles): coalesced reads, and
// writes in runs.
struct TagArgs {
  const int64_t *tag_off;
  const int32_t *tags;
  int64_t *tagcur;          // int64[ntiles * K]: scanned tile tag counts
  const int64_t *tag_base;  // int64[K + 1]: exclusive prefix of the buckets' tag totals
  int64_t *tag_off_out;
  int32_t *tags_out;
  int tcur_smem;            // the tag cursors fit in shared memory
};

// The stable scatter (see the file comment): chunks sorted by passes of B0
// and then B1 (0: none) digit bits.  perm_out[slot] = item index.
template <int B0, int B1, bool TAGS>
__global__ void __launch_bounds__(kPThreads, TAGS ? 1 : kPartTilesPerSM)
    part_scatter_kernel(const int32_t *__restrict__ labels, int64_t N, int K, int64_t tile,
                        const int32_t *__restrict__ tileoff, const int64_t *__restrict__ offsets,
                        int32_t *__restrict__ perm_out, TagArgs ta) {
  constexpr int BMAX = B0 > B1 ? B0 : B1;
  extern __shared__ uint32_t psm[];
  int32_t *cursor = reinterpret_cast<int32_t *>(psm);
  uint32_t *ka = psm + round4(K);
  uint32_t *kb = ka + kPartChunk;
  int32_t *wcnt = reinterpret_cast<int32_t *>(kb + kPartChunk);
  int32_t *wsum = reinterpret_cast<int32_t *>(psm + scatter_wsum_word(K, BMAX));
  // TAGS: per-(j, warp) segment sums of the tag-length scan, staged offsets,
  // destinations by item, tag cursors
  int64_t *segsum = reinterpret_cast<int64_t *>(psm + scatter_segsum_word(K, BMAX));
  int64_t *toff = reinterpret_cast<int64_t *>(psm + scatter_toff_word(K, BMAX));
  int64_t *dsts = toff + kPartChunk + 2;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t t = blockIdx.x;
  for (int k = threadIdx.x; k < K; k += kPThreads) cursor[k] = (int32_t)(offsets[k] + tileoff[t * K + k]);
  int64_t *tcur = nullptr;
  if (TAGS) {
    tcur = ta.tcur_smem ? dsts + kPartChunk : ta.tagcur + t * K;
    for (int k = threadIdx.x; k < K; k += kPThreads) tcur[k] = ta.tagcur[t * K + k] + ta.tag_base[k];
  }
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
    const int nvalid = (int)min((int64_t)kPartChunk, end - pos);
    if (TAGS) {
      // toff[p] = tag_off[pos + p], p <= nvalid (8-byte asynchronous copies)
      for (int q = threadIdx.x; q <= nvalid; q += kPThreads)
        asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(smem_u32(toff + q)), "l"(ta.tag_off + pos + q)
                     : "memory");
      asm volatile("cp.async.commit_group;" ::: "memory");
    }
    uint32_t v[kPR];
    unsigned okmask = 0;  // bit r: this thread's item r has a label in [0, K)
#pragma unroll
    for (int r = 0; r < kPR; ++r) {
      const bool ok = lab[r] >= 0 && lab[r] < K;
      const unsigned key = ok ? (unsigned)lab[r] : (unsigned)K;
      v[r] = (key << 16) | (unsigned)(pbase + 32 * r);
      if (ok) okmask |= 1u << r;
    }
    // the next chunk's labels are in flight during the sort of this one
    const int64_t nxt = pos + kPartChunk;
#pragma unroll
    for (int r = 0; r < kPR; ++r) {
      const int64_t i = nxt + pbase + 32 * r;
      lab[r] = i < end ? __ldg(labels + i) : -1;
    }
    rank_pass<B0, 0>(v, kb, wcnt, wsum);
    const uint32_t *sorted = kb;
    uint32_t *spare = ka;
    if (B1 > 0) {
      uint32_t w[kPR];
#pragma unroll
      for (int r = 0; r < kPR; ++r) w[r] = kb[pbase + 32 * r];
      rank_pass<(B1 > 0 ? B1 : 1), B0>(w, ka, wcnt, wsum);
      sorted = ka;
      spare = kb;
    }
    // runs of equal keys: the first item of a run turns the bucket's cursor
    // into its base (cursor - position), every item stores at base + position,
    // the last item moves the cursor past the run.  Sorted position q of item
    // j of this thread is tid + kPThreads j: consecutive lanes, consecutive q.
    uint32_t sv[kPR];
    unsigned last = 0;  // bit j: item j ends its run
#pragma unroll
    for (int j = 0; j < kPR; ++j) {
      const int q = threadIdx.x + kPThreads * j;
      sv[j] = sorted[q];
      const unsigned key = sv[j] >> 16;
      unsigned prev = __shfl_up_sync(0xffffffffu, key, 1);
      unsigned next = __shfl_down_sync(0xffffffffu, key, 1);
      if (lane == 0) prev = q > 0 ? (sorted[q - 1] >> 16) : 0xFFFFFFFFu;
      if (lane == 31) next = q + 1 < kPartChunk ? (sorted[q + 1] >> 16) : 0xFFFFFFFFu;
      if (key != next) last |= 1u << j;
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
      }
      if (TAGS) spare[q] = (uint32_t)slot[j];
    }
    __syncthreads();
#pragma unroll
    for (int j = 0; j < kPR; ++j)
      if (slot[j] >= 0 && ((last >> j) & 1u)) cursor[sv[j] >> 16] = slot[j] + 1;
    if (TAGS) {
      asm volatile("cp.async.wait_all;" ::: "memory");
      __syncthreads();
      // lengths in sorted order and their block-wide exclusive prefix: a warp
      // scan per j, then the 16 kPR (j, warp) segments in order
      int64_t incl[kPR];
      int32_t len[kPR];
      // 32-bit warp scans when the chunk's lists hold fewer than 2^31 tags
      const bool narrow = toff[nvalid] - toff[0] < ((int64_t)1 << 31);
#pragma unroll
      for (int j = 0; j < kPR; ++j) {
        const unsigned key = sv[j] >> 16;
        const int p = (int)(sv[j] & 0xFFFFu);
        len[j] = key < (unsigned)K ? (int32_t)(toff[p + 1] - toff[p]) : 0;
        int64_t x;
        if (narrow) {
          int xi = len[j];
#pragma unroll
          for (int o = 1; o < 32; o <<= 1) {
            const int u = __shfl_up_sync(0xffffffffu, xi, o);
            if (lane >= o) xi += u;
          }
          x = xi;
        } else {
          x = len[j];
#pragma unroll
          for (int o = 1; o < 32; o <<= 1) {
            const int64_t u = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x += u;
          }
        }
        incl[j] = x;
        if (lane == 31) segsum[j * kPWarps + warp] = x;
      }
      __syncthreads();
      if (warp == 0) {
        constexpr int NS = kPR * kPWarps;  // segments in sorted order
        constexpr int PS = NS / 32;
        int64_t sv4[PS];
        int64_t loc = 0;
#pragma unroll
        for (int u = 0; u < PS; ++u) {
          sv4[u] = segsum[lane * PS + u];
          loc += sv4[u];
        }
        int64_t x = loc;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int64_t u = __shfl_up_sync(0xffffffffu, x, o);
          if (lane >= o) x += u;
        }
        int64_t run = x - loc;
#pragma unroll
        for (int u = 0; u < PS; ++u) {
          segsum[lane * PS + u] = run;
          run += sv4[u];
        }
      }
      __syncthreads();
      // run starts: tag cursor -> base (cursor - P of the run's first item)
#pragma unroll
      for (int j = 0; j < kPR; ++j) {
        const int q = threadIdx.x + kPThreads * j;
        incl[j] += segsum[j * kPWarps + warp] - len[j];  // P: exclusive prefix of this item
        const unsigned key = sv[j] >> 16;
        unsigned prev = __shfl_up_sync(0xffffffffu, key, 1);
        if (lane == 0) prev = q > 0 ? (sorted[q - 1] >> 16) : 0xFFFFFFFFu;
        if (key < (unsigned)K && key != prev) tcur[key] -= incl[j];
      }
      __syncthreads();
      // destinations: by slot (tag_off_out) and by item (for the copy)
#pragma unroll
      for (int j = 0; j < kPR; ++j) {
        const int q = threadIdx.x + kPThreads * j;
        const unsigned key = sv[j] >> 16;
        if (key < (unsigned)K) {
          const int64_t dst = tcur[key] + incl[j];
          ta.tag_off_out[(int32_t)spare[q]] = dst;
          dsts[sv[j] & 0xFFFFu] = dst;
          incl[j] = dst + len[j];  // the end of this item's list
        }
      }
      __syncthreads();
#pragma unroll
      for (int j = 0; j < kPR; ++j)
        if ((sv[j] >> 16) < (unsigned)K && ((last >> j) & 1u)) tcur[sv[j] >> 16] = incl[j];
      // copy in source order: item r of this thread sits at pbase + 32 r, so
      // a warp's loads of its lists' first tags read neighbouring memory; the
      // first four tags of two items are loaded before any is stored (eight
      // loads in flight), longer lists finish in a loop
#pragma unroll 1
      for (int r = 0; r < kPR; r += 2) {
        int64_t src[2], dst[2];
        int32_t ln[2], v[2][4];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int pp = pbase + 32 * (r + h);
          const bool ok = (okmask >> (r + h)) & 1u;
          src[h] = ok ? toff[pp] : 0;
          ln[h] = ok ? (int32_t)(toff[pp + 1] - src[h]) : 0;
          dst[h] = ok ? dsts[pp] : 0;
#pragma unroll
          for (int u = 0; u < 4; ++u) v[h][u] = u < ln[h] ? __ldg(ta.tags + src[h] + u) : 0;
        }
#pragma unroll
        for (int h = 0; h < 2; ++h) {
#pragma unroll
          for (int u = 0; u < 4; ++u)
            if (u < ln[h]) ta.tags_out[dst[h] + u] = v[h][u];
          for (int32_t u = 4; u < ln[h]; ++u) ta.tags_out[dst[h] + u] = __ldg(ta.tags + src[h] + u);
        }
      }
      __syncthreads();  // toff and dsts are rewritten for the next chunk
    }
    // the next chunk's first rank pass synchronises before its key buffers are reused
  }
}

// tag_off_out[s] = the total of the moved lists for the slots past the valid
// items, s in [offsets[K], N] (tag_off_out[N] at least).
__global__ void part_tag_tail_kernel(const int64_t *__restrict__ offsets, int K, int64_t N,
                                     const int64_t *__restrict__ tag_base, int64_t *__restrict__ tag_off_out) {
  const int64_t total = tag_base[K];
  for (int64_t s = offsets[K] + (int64_t)blockIdx.x * blockDim.x + threadIdx.x; s <= N;
       s += (int64_t)gridDim.x * blockDim.x)
    tag_off_out[s] = total;
}

using ScatterFn = void (*)(const int32_t *, int64_t, int, int64_t, const int32_t *, const int64_t *, int32_t *,
                           TagArgs);

// sorted_labels[s] = the bucket of slot s (offsets[k] <= s < offsets[k+1]),
// for s < offsets[K]: every thread fills 16 consecutive slots, finding the
// bucket of its first slot by binary search and stepping over the buckets
// that end inside its slots; 16-byte stores.
constexpr int kFillSlots = 16;
__global__ void part_fill_labels_kernel(const int64_t *__restrict__ offsets, int K, int64_t N,
                                        int32_t *__restrict__ sorted_labels) {
  const int64_t s0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) * kFillSlots;
  const int64_t n = __ldg(offsets + K);
  if (s0 >= n || s0 >= N) return;
  int lo = 0, hi = K - 1;  // the largest k with offsets[k] <= s0
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (__ldg(offsets + mid) <= s0)
      lo = mid;
    else
      hi = mid - 1;
  }
  int k = lo;
  int64_t next = __ldg(offsets + k + 1);
  int32_t v[kFillSlots];
#pragma unroll
  for (int u = 0; u < kFillSlots; ++u) {
    while (s0 + u >= next && k + 1 < K) next = __ldg(offsets + (++k) + 1);
    v[u] = k;
  }
  const int64_t m = min((int64_t)kFillSlots, n - s0);
  if (m == kFillSlots && (reinterpret_cast<uintptr_t>(sorted_labels + s0) & 15u) == 0) {
    int4 *d = reinterpret_cast<int4 *>(sorted_labels + s0);
#pragma unroll
    for (int u = 0; u < kFillSlots / 4; ++u) d[u] = make_int4(v[4 * u], v[4 * u + 1], v[4 * u + 2], v[4 * u + 3]);
  } else {
    for (int u = 0; u < m; ++u) sorted_labels[s0 + u] = v[u];
  }
}

// The scatter instance for digit bits (b0, b1): one pass of 1 .. 8 bits, or
// two passes of 4 .. 8 bits (keys of 9 .. 15 bits).
template <bool TAGS>
ScatterFn scatter_fn(int b0, int b1) {
  switch (b0 * 16 + b1) {
    case 1 * 16: return part_scatter_kernel<1, 0, TAGS>;
    case 2 * 16: return part_scatter_kernel<2, 0, TAGS>;
    case 3 * 16: return part_scatter_kernel<3, 0, TAGS>;
    case 4 * 16: return part_scatter_kernel<4, 0, TAGS>;
    case 5 * 16: return part_scatter_kernel<5, 0, TAGS>;
    case 6 * 16: return part_scatter_kernel<6, 0, TAGS>;
    case 7 * 16: return part_scatter_kernel<7, 0, TAGS>;
    case 8 * 16: return part_scatter_kernel<8, 0, TAGS>;
    case 4 * 16 + 5: return part_scatter_kernel<4, 5, TAGS>;
    case 5 * 16 + 5: return part_scatter_kernel<5, 5, TAGS>;
    case 5 * 16 + 6: return part_scatter_kernel<5, 6, TAGS>;
    case 6 * 16 + 6: return part_scatter_kernel<6, 6, TAGS>;
    case 6 * 16 + 7: return part_scatter_kernel<6, 7, TAGS>;
    case 7 * 16 + 7: return part_scatter_kernel<7, 7, TAGS>;
    case 7 * 16 + 8: return part_scatter_kernel<7, 8, TAGS>;
    default: return nullptr;
  }
}

}  // namespace

PartLayout part_layout(size_t base, int64_t N, int K, bool tags) {
  PartLayout pl;
  int bits = 0;
  while ((1 << bits) < K + 1) ++bits;  // labels 0 .. K-1 and the key K of an invalid label
  pl.b0 = bits <= kMaxDigitBits ? bits : bits / 2;
  pl.b1 = bits - pl.b0;
  // two CTAs per SM; one with tag lists (whose scatter needs more registers)
  const int64_t target = (tags ? 1 : kPartTilesPerSM) * kPartSMs;
  int64_t tile = (N + target - 1) / target;
  tile = (tile + kPartChunk - 1) / kPartChunk * kPartChunk;
  if (tile < kPartChunk) tile = kPartChunk;
  pl.tile = tile;
  pl.ntiles = N > 0 ? (N + tile - 1) / tile : 0;
  const size_t nt = (size_t)(pl.ntiles > 0 ? pl.ntiles : 1);
  size_t off = align_up(base, 256);
  pl.tilecnt = off;
  off = align_up(off + nt * K * sizeof(int32_t), 256);
  pl.hist = off;
  off = align_up(off + (size_t)K * sizeof(int64_t), 256);
  pl.offs = off;
  off = align_up(off + (size_t)(K + 1) * sizeof(int64_t), 256);
  pl.tagcnt = pl.tag_hist = pl.tag_base = 0;
  if (tags) {
    pl.tagcnt = off;
    off = align_up(off + nt * K * sizeof(int64_t), 256);
    pl.tag_hist = off;
    off = align_up(off + (size_t)K * sizeof(int64_t), 256);
    pl.tag_base = off;
    off = align_up(off + (size_t)(K + 1) * sizeof(int64_t), 256);
  }
  pl.end = off;
  return pl;
}

cudaError_t launch_partition(const int32_t *labels, int64_t N, int K, const PartLayout &pl, char *ws,
                             int64_t *hist, int64_t *offsets, int32_t *perm, int32_t *sorted_labels, Header *hdr,
                             cudaStream_t s, const TagLists *tl) {
  const bool tags = tl != nullptr;
  if (tags && !pl.tagcnt) return cudaErrorInvalidValue;
  int32_t *tilecnt = reinterpret_cast<int32_t *>(ws + pl.tilecnt);
  int64_t *tagcnt = tags ? reinterpret_cast<int64_t *>(ws + pl.tagcnt) : nullptr;
  int64_t *tag_hist = tags ? reinterpret_cast<int64_t *>(ws + pl.tag_hist) : nullptr;
  int64_t *tag_base = tags ? reinterpret_cast<int64_t *>(ws + pl.tag_base) : nullptr;
  const size_t smc = (size_t)round4(K) * sizeof(int32_t) + (tags ? (size_t)K * sizeof(int64_t) : 0);
  const int bmax = pl.b0 > pl.b1 ? pl.b0 : pl.b1;
  const bool tcur_smem = tags && scatter_smem_words(K, bmax, true, true) * sizeof(uint32_t) <= kMaxSmemScatter;
  const size_t sms = scatter_smem_words(K, bmax, tags, tcur_smem) * sizeof(uint32_t);
  auto count = tags ? part_count_kernel<true> : part_count_kernel<false>;
  ScatterFn scatter = tags ? scatter_fn<true>(pl.b0, pl.b1) : scatter_fn<false>(pl.b0, pl.b1);
  if (!scatter) return cudaErrorInvalidValue;
  cudaError_t e;
  if (smc > 48 * 1024) {
    e = cudaFuncSetAttribute(count, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smc);
    if (e != cudaSuccess) return e;
  }
  if (sms > 48 * 1024) {
    e = cudaFuncSetAttribute(scatter, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sms);
    if (e != cudaSuccess) return e;
  }
  if (pl.ntiles > 0) {
    count<<<(unsigned)pl.ntiles, kPThreads, smc, s>>>(labels, N, K, pl.tile, tilecnt, tags ? tl->tag_off : nullptr,
                                                      tagcnt, hdr);
    count_launch();
  }
  part_colscan_kernel<int32_t><<<(K + 31) / 32, 1024, 0, s>>>(tilecnt, pl.ntiles, K, hist);
  part_offsets_kernel<<<1, 1024, 0, s>>>(hist, K, offsets);
  count_launch(2);
  if (tags) {
    part_colscan_kernel<int64_t><<<(K + 31) / 32, 1024, 0, s>>>(tagcnt, pl.ntiles, K, tag_hist);
    part_offsets_kernel<<<1, 1024, 0, s>>>(tag_hist, K, tag_base);
    count_launch(2);
  }
  if (pl.ntiles > 0) {
    TagArgs ta{};
    if (tags) ta = TagArgs{tl->tag_off, tl->tags, tagcnt, tag_base, tl->tag_off_out, tl->tags_out, tcur_smem ? 1 : 0};
    scatter<<<(unsigned)pl.ntiles, kPThreads, sms, s>>>(labels, N, K, pl.tile, tilecnt, offsets, perm, ta);
    count_launch();
    if (sorted_labels) {
      const int64_t threads = (N + kFillSlots - 1) / kFillSlots;
      part_fill_labels_kernel<<<(unsigned)((threads + 255) / 256), 256, 0, s>>>(offsets, K, N, sorted_labels);
      count_launch();
    }
  }
  if (tags) {
    part_tag_tail_kernel<<<8, 256, 0, s>>>(offsets, K, N, tag_base, tl->tag_off_out);
    count_launch();
  }
  return cudaGetLastError();
}

}  // namespace hme
