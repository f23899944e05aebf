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
//   4. scatter  each CTA walks its tile in index order, kPartChunk items at
//               a time.  A chunk is sorted by label inside shared memory with
//               a stable least-significant-digit radix sort of one or two
//               passes (digits of at most 7 bits, 8 for the last pass of
//               15-bit keys; every thread counts its 16 consecutive items per
//               digit in private 16-bit counters and one block-wide scan of
//               the counters gives every item its place), so that items of a
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

#include <algorithm>

#ifndef HME_PART_MAXB
#define HME_PART_MAXB 5
#endif

namespace hme {

namespace {

constexpr int kPThreads = 512;                // threads of a count CTA
constexpr int kSThreads = 512;                // threads of a scatter CTA
constexpr int kSWarps = kSThreads / 32;
constexpr int kSR = kPartChunk / kSThreads;   // items per scatter thread per chunk
constexpr int kMaxDigitBits = HME_PART_MAXB;
constexpr int kPartTilesPerSM = 2;
constexpr int kPartWideK = 2048;             // from this K on, one tile per SM
constexpr int kPartSMs = 152;                 // GB300: the tile count fills two CTAs per SM
constexpr size_t kMaxSmemScatter = 227 * 1024;
static_assert(kPartChunk % kSThreads == 0 && kPartChunk <= 65536, "chunk positions fit 16 bits");
static_assert(kSR <= 16 && kPartChunk < 65536, "per-thread digit counts and prefixes fit 16-bit halves");

__host__ __device__ __forceinline__ int round4(int k) { return (k + 3) / 4 * 4; }

// Counter words of a rank pass of B digit bits: two 16-bit counters per word,
// 2^B / 2 words per thread, laid out word-lane-major (word lane l of thread t
// at l * kSThreads + t) with one padding word after every raking segment of
// 2^B / 2 words (the segments are then read without bank conflicts).
__host__ __device__ constexpr int ctr_lanes(int B) { return B >= 1 ? (1 << B) / 2 : 1; }
__host__ __device__ __forceinline__ size_t ctr_words(int bmax) {
  return (size_t)ctr_lanes(bmax) * kSThreads + kSThreads;
}

// Shared-memory layout of the scatter CTA, in 32-bit words: cursors, the key
// buffer, the rank counters, the scan's warp totals; with tag lists then the
// slot of every sorted position, the (j, warp) segment sums of the tag-length
// scan (int64), the chunk's staged tag offsets int64[kPartChunk + 1], the
// list destinations by item int64[kPartChunk] and (when it fits) the tag
// cursors int64[K], the int64 arrays from an even word.
// Key buffer: position i at word i + i / 32, so that both a thread's 16
// consecutive positions (blocked) and a warp's 32 consecutive positions
// (strided) fall into distinct banks.
__host__ __device__ __forceinline__ int kpad(int i) { return i + (i >> 5); }
__host__ __device__ __forceinline__ size_t scatter_ctr_word(int K) {
  return (size_t)round4(K) + (size_t)kPartChunk + kPartChunk / 32;
}
__host__ __device__ __forceinline__ size_t scatter_wsum_word(int K, int bmax) {
  return scatter_ctr_word(K) + ctr_words(bmax);
}
__host__ __device__ __forceinline__ size_t scatter_spare_word(int K, int bmax) {
  return scatter_wsum_word(K, bmax) + 32;
}
__host__ __device__ __forceinline__ size_t scatter_segsum_word(int K, int bmax) {
  return (scatter_spare_word(K, bmax) + kPartChunk + 1) & ~(size_t)1;
}
__host__ __device__ __forceinline__ size_t scatter_toff_word(int K, int bmax) {
  return scatter_segsum_word(K, bmax) + 2 * (size_t)kSR * kSWarps;
}
__host__ __device__ __forceinline__ size_t scatter_smem_words(int K, int bmax, bool tags = false,
                                                             bool tcur_smem = false) {
  if (!tags) return scatter_spare_word(K, bmax);
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

// One stable counting pass of the block-local radix sort, without ballots:
// every thread keeps private counters.  Thread t holds the kSR consecutive
// items kSR t .. kSR t + kSR - 1 of the current order; item r has packed value
// v[r] = key << 16 | (position in the chunk's index order) and digit
// (key >> SHIFT) mod 2^B.  (1) Each thread counts its items per digit, an
// item's rank among its thread's items of the same digit being the count
// before it (16-bit counters, two per word: digits l and l + 2^B/2 in word
// lane l).  (2) An exclusive scan of the words in (word lane, thread) order
// -- each thread sums its raking segment, one block scan of the segment sums
// -- gives, in each half, the items of smaller digit or of the same digit in
// lower threads; the upper halves then add the count of all lower-half
// digits.  (3) Every item is written to out[its digit-and-thread prefix +
// its rank] (padded index, kpad), its place in the order by (digit, current
// position).
template <int B, int SHIFT>
__device__ __forceinline__ void rank_pass(const uint32_t (&v)[kSR], uint32_t *out, uint32_t *ctr, uint32_t *wsum) {
  constexpr int CL = ctr_lanes(B);   // counter words per thread
  constexpr int SEG = CL;            // raking segment of a thread (words)
  constexpr unsigned DMASK = (1u << B) - 1u;
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  uint32_t *seg = ctr + t * (SEG + 1);  // this thread's raking segment (padded layout)
#pragma unroll
  for (int u = 0; u < SEG; ++u) seg[u] = 0;
  __syncthreads();
  uint32_t at[kSR];  // padded word index << 5 | half shift
  uint32_t rk[kSR];
#pragma unroll
  for (int r = 0; r < kSR; ++r) {
    const unsigned d = (v[r] >> (16 + SHIFT)) & DMASK;
    const unsigned l = d % CL, sh = (d / CL) * 16;
    const unsigned i = l * kSThreads + t;
    const unsigned pi = i + i / SEG;
    // a shared atomic, not a load and a store: the thread's 16 increments
    // then issue back to back (only this thread touches these words)
    const uint32_t w = atomicAdd(&ctr[pi], 1u << sh);
    rk[r] = (w >> sh) & 0xFFFFu;
    at[r] = (pi << 5) | sh;
  }
  __syncthreads();
  // raking: segment sums, block exclusive scan (packed 16-bit halves)
  uint32_t sum = 0;
#pragma unroll
  for (int u = 0; u < SEG; ++u) sum += seg[u];
  uint32_t incl = sum;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t x = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += x;
  }
  if (lane == 31) wsum[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    const uint32_t w = lane < kSWarps ? wsum[lane] : 0u;
    uint32_t wi = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t x = __shfl_up_sync(0xffffffffu, wi, o);
      if (lane >= o) wi += x;
    }
    if (lane < kSWarps) wsum[lane] = wi - w;
    if (lane == kSWarps - 1) wsum[kSWarps] = wi;  // the grand total
  }
  __syncthreads();
  // the upper halves follow every lower-half digit
  uint32_t run = wsum[warp] + incl - sum + ((wsum[kSWarps] & 0xFFFFu) << 16);
#pragma unroll
  for (int u = 0; u < SEG; ++u) {
    const uint32_t w = seg[u];
    seg[u] = run;
    run += w;
  }
  __syncthreads();
#pragma unroll
  for (int r = 0; r < kSR; ++r) {
    const uint32_t w = ctr[at[r] >> 5];
    out[kpad((int)(((w >> (at[r] & 31u)) & 0xFFFFu) + rk[r]))] = v[r];
  }
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

// The stable scatter (see the file comment): chunks sorted by passes of B0,
// then B1 and B2 (0: none) digit bits.  perm_out[slot] = item index.
template <int B0, int B1, int B2, bool TAGS>
__global__ void __launch_bounds__(kSThreads, TAGS ? 1 : kPartTilesPerSM)
    part_scatter_kernel(const int32_t *__restrict__ labels, int64_t N, int K, int64_t tile,
                        const int32_t *__restrict__ tileoff, const int64_t *__restrict__ offsets,
                        int32_t *__restrict__ perm_out, TagArgs ta, int64_t *__restrict__ fz_hist,
                        int64_t *__restrict__ fz_offs, Header *hdr) {
  constexpr int BMAX = B0 > B1 ? (B0 > B2 ? B0 : B2) : (B1 > B2 ? B1 : B2);
  extern __shared__ uint32_t psm[];
  int32_t *cursor = reinterpret_cast<int32_t *>(psm);
  uint32_t *keys = psm + round4(K);
  uint32_t *ctr = psm + scatter_ctr_word(K);
  uint32_t *wsum = psm + scatter_wsum_word(K, BMAX);
  // TAGS: slot by sorted position, per-(j, warp) segment sums of the tag-length
  // scan, staged offsets, destinations by item, tag cursors
  uint32_t *spare = psm + scatter_spare_word(K, BMAX);
  int64_t *segsum = reinterpret_cast<int64_t *>(psm + scatter_segsum_word(K, BMAX));
  int64_t *toff = reinterpret_cast<int64_t *>(psm + scatter_toff_word(K, BMAX));
  int64_t *dsts = toff + kPartChunk + 2;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t t = blockIdx.x;
  if (fz_offs) {
    // one tile holds every item (no TAGS): count it here, and the exclusive
    // prefix of the counts is both offsets and the cursors
    for (int k = threadIdx.x; k < K; k += kSThreads) cursor[k] = 0;
    __syncthreads();
    bool bad = false;
    for (int64_t i = threadIdx.x; i < N; i += kSThreads) {
      const int v = __ldg(labels + i);
      if (v >= 0 && v < K)
        atomicAdd(&cursor[v], 1);
      else
        bad = true;
    }
    if (bad) atomicOr(&hdr->status, (uint32_t)kStatusBadLabel);
    __syncthreads();
    const int per = (K + kSThreads - 1) / kSThreads;
    const int k0 = min(K, (int)threadIdx.x * per), k1 = min(K, k0 + per);
    int32_t loc = 0;
    for (int k = k0; k < k1; ++k) loc += cursor[k];
    int32_t incl = loc;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int32_t x = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += x;
    }
    if (lane == 31) wsum[warp] = (uint32_t)incl;
    __syncthreads();
    if (warp == 0) {
      const int32_t x0 = lane < kSWarps ? (int32_t)wsum[lane] : 0;
      int32_t xi = x0;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int32_t x = __shfl_up_sync(0xffffffffu, xi, o);
        if (lane >= o) xi += x;
      }
      if (lane < kSWarps) wsum[lane] = (uint32_t)(xi - x0);
    }
    __syncthreads();
    int32_t run = (int32_t)wsum[warp] + incl - loc;
    for (int k = k0; k < k1; ++k) {
      const int32_t c = cursor[k];
      fz_hist[k] = c;
      fz_offs[k] = run;
      cursor[k] = run;
      run += c;
    }
    if (threadIdx.x == kSThreads - 1) fz_offs[K] = run;
    __syncthreads();
  } else {
    for (int k = threadIdx.x; k < K; k += kSThreads) cursor[k] = (int32_t)(offsets[k] + tileoff[t * K + k]);
  }
  int64_t *tcur = nullptr;
  if (TAGS) {
    tcur = ta.tcur_smem ? dsts + kPartChunk : ta.tagcur + t * K;
    for (int k = threadIdx.x; k < K; k += kSThreads) tcur[k] = ta.tagcur[t * K + k] + ta.tag_base[k];
  }
  const int64_t start = t * tile;
  const int64_t end = min(N, start + tile);
  // thread t holds chunk positions kSR t .. kSR t + kSR - 1 (blocked); the
  // base is 16-byte aligned when labels is (start is a multiple of the chunk)
  const int pbase = threadIdx.x * kSR;
  const bool vec = (reinterpret_cast<uintptr_t>(labels) & 15u) == 0;
  int32_t lab[kSR];
  auto load = [&](int64_t at) {
    if (vec && at + pbase + kSR <= end) {
      const int4 *src = reinterpret_cast<const int4 *>(labels + at + pbase);
#pragma unroll
      for (int u = 0; u < kSR / 4; ++u) {
        const int4 x = __ldg(src + u);
        lab[4 * u] = x.x;
        lab[4 * u + 1] = x.y;
        lab[4 * u + 2] = x.z;
        lab[4 * u + 3] = x.w;
      }
    } else {
#pragma unroll
      for (int r = 0; r < kSR; ++r) {
        const int64_t i = at + pbase + r;
        lab[r] = i < end ? __ldg(labels + i) : -1;
      }
    }
  };
  load(start);
  for (int64_t pos = start; pos < end; pos += kPartChunk) {
    const int nvalid = (int)min((int64_t)kPartChunk, end - pos);
    if (TAGS) {
      // toff[p] = tag_off[pos + p], p <= nvalid (8-byte asynchronous copies)
      for (int q = threadIdx.x; q <= nvalid; q += kSThreads)
        asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(smem_u32(toff + q)), "l"(ta.tag_off + pos + q)
                     : "memory");
      asm volatile("cp.async.commit_group;" ::: "memory");
    }
    uint32_t v[kSR];
#pragma unroll
    for (int r = 0; r < kSR; ++r) {
      const unsigned key = (lab[r] >= 0 && lab[r] < K) ? (unsigned)lab[r] : (unsigned)K;
      v[r] = (key << 16) | (unsigned)(pbase + r);
    }
    // the next chunk's labels are in flight during the sort of this one
    load(pos + kPartChunk);
    rank_pass<B0, 0>(v, keys, ctr, wsum);
    if (B1 > 0) {  // the second pass reads its items before the first writes over them (rank_pass syncs)
#pragma unroll
      for (int r = 0; r < kSR; ++r) v[r] = keys[kpad(pbase + r)];
      rank_pass<(B1 > 0 ? B1 : 1), B0>(v, keys, ctr, wsum);
    }
    if (B2 > 0) {
#pragma unroll
      for (int r = 0; r < kSR; ++r) v[r] = keys[kpad(pbase + r)];
      rank_pass<(B2 > 0 ? B2 : 1), B0 + B1>(v, keys, ctr, wsum);
    }
    const uint32_t *sorted = keys;
    // runs of equal keys: the first item of a run turns the bucket's cursor
    // into its base (cursor - position), every item stores at base + position,
    // the last item moves the cursor past the run.  Sorted position q of item
    // j of this thread is tid + kSThreads j: consecutive lanes, consecutive q.
    uint32_t sv[kSR];
    unsigned last = 0;  // bit j: item j ends its run
#pragma unroll
    for (int j = 0; j < kSR; ++j) {
      const int q = threadIdx.x + kSThreads * j;
      sv[j] = sorted[kpad(q)];
      const unsigned key = sv[j] >> 16;
      unsigned prev = __shfl_up_sync(0xffffffffu, key, 1);
      unsigned next = __shfl_down_sync(0xffffffffu, key, 1);
      if (lane == 0) prev = q > 0 ? (sorted[kpad(q - 1)] >> 16) : 0xFFFFFFFFu;
      if (lane == 31) next = q + 1 < kPartChunk ? (sorted[kpad(q + 1)] >> 16) : 0xFFFFFFFFu;
      if (key != next) last |= 1u << j;
      if (key < (unsigned)K && key != prev) cursor[key] -= q;
    }
    __syncthreads();
    int32_t slot[kSR];
#pragma unroll
    for (int j = 0; j < kSR; ++j) {
      const int q = threadIdx.x + kSThreads * j;
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
    for (int j = 0; j < kSR; ++j)
      if (slot[j] >= 0 && ((last >> j) & 1u)) cursor[sv[j] >> 16] = slot[j] + 1;
    if (TAGS) {
      asm volatile("cp.async.wait_all;" ::: "memory");
      __syncthreads();
      // lengths in sorted order and their block-wide exclusive prefix: a warp
      // scan per j, then the kSR kSWarps (j, warp) segments in order
      int64_t incl[kSR];
      int32_t len[kSR];
      // 32-bit warp scans when the chunk's lists hold fewer than 2^31 tags
      const bool narrow = toff[nvalid] - toff[0] < ((int64_t)1 << 31);
#pragma unroll
      for (int j = 0; j < kSR; ++j) {
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
        if (lane == 31) segsum[j * kSWarps + warp] = x;
      }
      __syncthreads();
      if (warp == 0) {
        constexpr int NS = kSR * kSWarps;  // segments in sorted order
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
      for (int j = 0; j < kSR; ++j) {
        const int q = threadIdx.x + kSThreads * j;
        incl[j] += segsum[j * kSWarps + warp] - len[j];  // P: exclusive prefix of this item
        const unsigned key = sv[j] >> 16;
        unsigned prev = __shfl_up_sync(0xffffffffu, key, 1);
        if (lane == 0) prev = q > 0 ? (sorted[kpad(q - 1)] >> 16) : 0xFFFFFFFFu;
        if (key < (unsigned)K && key != prev) tcur[key] -= incl[j];
      }
      __syncthreads();
      // destinations: by slot (tag_off_out) and by item (for the copy; -1:
      // an invalid label or a position past the tile, whose list stays)
#pragma unroll
      for (int j = 0; j < kSR; ++j) {
        const int q = threadIdx.x + kSThreads * j;
        const unsigned key = sv[j] >> 16;
        if (key < (unsigned)K) {
          const int64_t dst = tcur[key] + incl[j];
          ta.tag_off_out[(int32_t)spare[q]] = dst;
          dsts[sv[j] & 0xFFFFu] = dst;
          incl[j] = dst + len[j];  // the end of this item's list
        } else {
          dsts[sv[j] & 0xFFFFu] = -1;
        }
      }
      __syncthreads();
#pragma unroll
      for (int j = 0; j < kSR; ++j)
        if ((sv[j] >> 16) < (unsigned)K && ((last >> j) & 1u)) tcur[sv[j] >> 16] = incl[j];
      // copy in source order: item p = tid + kSThreads j, so a warp's loads of
      // its lists' first tags read neighbouring memory; the first four tags of
      // two items are loaded before any is stored (eight loads in flight),
      // longer lists finish in a loop
#pragma unroll 1
      for (int j = 0; j < kSR; j += 2) {
        int64_t src[2], dst[2];
        int32_t ln[2], w[2][4];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int pp = threadIdx.x + kSThreads * (j + h);
          dst[h] = dsts[pp];
          const bool ok = dst[h] >= 0;
          src[h] = ok ? toff[pp] : 0;
          ln[h] = ok ? (int32_t)(toff[pp + 1] - src[h]) : 0;
#pragma unroll
          for (int u = 0; u < 4; ++u) w[h][u] = u < ln[h] ? __ldg(ta.tags + src[h] + u) : 0;
        }
#pragma unroll
        for (int h = 0; h < 2; ++h) {
#pragma unroll
          for (int u = 0; u < 4; ++u)
            if (u < ln[h]) ta.tags_out[dst[h] + u] = w[h][u];
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
                           TagArgs, int64_t *, int64_t *, Header *);

// sorted_labels[s] = the bucket of slot s (offsets[k] <= s < offsets[k+1]),
// for s < offsets[K]: every thread finds the buckets of 16 consecutive slots
// (a binary search for the first, then a walk over the buckets that end
// inside them) and leaves them in shared memory; the block then stores its
// 4096 slots with consecutive threads on consecutive 16-byte words.
constexpr int kFillSlots = 16;
constexpr int kFillThreads = 256;
__global__ void __launch_bounds__(kFillThreads) part_fill_labels_kernel(const int64_t *__restrict__ offsets, int K,
                                                                        int64_t N, int32_t *__restrict__ sorted_labels) {
  __shared__ int32_t buf[kFillThreads * kFillSlots + kFillThreads];  // thread t's slots at t * 17
  const int64_t n = min(N, __ldg(offsets + K));
  const int64_t b0 = (int64_t)blockIdx.x * kFillThreads * kFillSlots;
  const int64_t s0 = b0 + (int64_t)threadIdx.x * kFillSlots;
  if (s0 < n) {
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
#pragma unroll
    for (int u = 0; u < kFillSlots; ++u) {
      while (s0 + u >= next && k + 1 < K) next = __ldg(offsets + (++k) + 1);
      buf[threadIdx.x * (kFillSlots + 1) + u] = k;
    }
  }
  __syncthreads();
  const int64_t m = min((int64_t)kFillThreads * kFillSlots, n - b0);  // slots of this block
  if (m <= 0) return;
  if (m == (int64_t)kFillThreads * kFillSlots && (reinterpret_cast<uintptr_t>(sorted_labels + b0) & 15u) == 0) {
#pragma unroll
    for (int u = 0; u < kFillSlots / 4; ++u) {
      const int w = (u * kFillThreads + threadIdx.x) * 4;  // first of four slots
      const int32_t *src = buf + (w / kFillSlots) * (kFillSlots + 1) + (w % kFillSlots);
      reinterpret_cast<int4 *>(sorted_labels + b0)[u * kFillThreads + threadIdx.x] =
          make_int4(src[0], src[1], src[2], src[3]);
    }
  } else {
    for (int w = threadIdx.x; w < m; w += kFillThreads)
      sorted_labels[b0 + w] = buf[(w / kFillSlots) * (kFillSlots + 1) + (w % kFillSlots)];
  }
}

// The scatter instance for digit bits (b0, b1, b2) (0: no such pass).
template <bool TAGS>
ScatterFn scatter_fn(int b0, int b1, int b2) {
  switch (b0 * 256 + b1 * 16 + b2) {
    case 1 * 256 + 0 * 16 + 0: return part_scatter_kernel<1, 0, 0, TAGS>;
    case 2 * 256 + 0 * 16 + 0: return part_scatter_kernel<2, 0, 0, TAGS>;
    case 3 * 256 + 0 * 16 + 0: return part_scatter_kernel<3, 0, 0, TAGS>;
    case 4 * 256 + 0 * 16 + 0: return part_scatter_kernel<4, 0, 0, TAGS>;
    case 5 * 256 + 0 * 16 + 0: return part_scatter_kernel<5, 0, 0, TAGS>;
    case 6 * 256 + 0 * 16 + 0: return part_scatter_kernel<6, 0, 0, TAGS>;
    case 7 * 256 + 0 * 16 + 0: return part_scatter_kernel<7, 0, 0, TAGS>;
    case 1 * 256 + 1 * 16 + 0: return part_scatter_kernel<1, 1, 0, TAGS>;
    case 2 * 256 + 1 * 16 + 0: return part_scatter_kernel<2, 1, 0, TAGS>;
    case 2 * 256 + 2 * 16 + 0: return part_scatter_kernel<2, 2, 0, TAGS>;
    case 3 * 256 + 2 * 16 + 0: return part_scatter_kernel<3, 2, 0, TAGS>;
    case 3 * 256 + 3 * 16 + 0: return part_scatter_kernel<3, 3, 0, TAGS>;
    case 4 * 256 + 3 * 16 + 0: return part_scatter_kernel<4, 3, 0, TAGS>;
    case 4 * 256 + 4 * 16 + 0: return part_scatter_kernel<4, 4, 0, TAGS>;
    case 5 * 256 + 4 * 16 + 0: return part_scatter_kernel<5, 4, 0, TAGS>;
    case 5 * 256 + 5 * 16 + 0: return part_scatter_kernel<5, 5, 0, TAGS>;
    case 6 * 256 + 5 * 16 + 0: return part_scatter_kernel<6, 5, 0, TAGS>;
    case 6 * 256 + 6 * 16 + 0: return part_scatter_kernel<6, 6, 0, TAGS>;
    case 7 * 256 + 6 * 16 + 0: return part_scatter_kernel<7, 6, 0, TAGS>;
    case 7 * 256 + 7 * 16 + 0: return part_scatter_kernel<7, 7, 0, TAGS>;
    case 1 * 256 + 1 * 16 + 1: return part_scatter_kernel<1, 1, 1, TAGS>;
    case 2 * 256 + 1 * 16 + 1: return part_scatter_kernel<2, 1, 1, TAGS>;
    case 2 * 256 + 2 * 16 + 1: return part_scatter_kernel<2, 2, 1, TAGS>;
    case 2 * 256 + 2 * 16 + 2: return part_scatter_kernel<2, 2, 2, TAGS>;
    case 3 * 256 + 2 * 16 + 2: return part_scatter_kernel<3, 2, 2, TAGS>;
    case 3 * 256 + 3 * 16 + 2: return part_scatter_kernel<3, 3, 2, TAGS>;
    case 3 * 256 + 3 * 16 + 3: return part_scatter_kernel<3, 3, 3, TAGS>;
    case 4 * 256 + 3 * 16 + 3: return part_scatter_kernel<4, 3, 3, TAGS>;
    case 4 * 256 + 4 * 16 + 3: return part_scatter_kernel<4, 4, 3, TAGS>;
    case 4 * 256 + 4 * 16 + 4: return part_scatter_kernel<4, 4, 4, TAGS>;
    case 5 * 256 + 4 * 16 + 4: return part_scatter_kernel<5, 4, 4, TAGS>;
    case 5 * 256 + 5 * 16 + 4: return part_scatter_kernel<5, 5, 4, TAGS>;
    case 5 * 256 + 5 * 16 + 5: return part_scatter_kernel<5, 5, 5, TAGS>;
    default: return nullptr;
  }
}

}  // namespace

PartLayout part_layout(size_t base, int64_t N, int K, bool tags) {
  PartLayout pl;
  int bits = 0;
  while ((1 << bits) < K + 1) ++bits;  // labels 0 .. K-1 and the key K of an invalid label
  // passes of at most kMaxDigitBits bits, as equal as possible (larger first):
  // small digits keep the per-thread counters, which every pass clears and
  // scans, small
  const int npass = (bits + kMaxDigitBits - 1) / kMaxDigitBits;
  int b[3] = {0, 0, 0};
  for (int i = 0; i < npass; ++i) b[i] = bits / npass + (i < bits % npass ? 1 : 0);
  pl.b0 = b[0];
  pl.b1 = b[1];
  pl.b2 = b[2];
  // two CTAs per SM; one with tag lists (whose scatter needs more registers)
  // or with K >= 2048, where the ntiles x K partly written output lines of
  // two tiles per SM no longer fit L2 (with labels spread over the buckets,
  // runs are about one item long and every store would reach DRAM as a
  // partial sector)
  const int64_t target = (tags || K >= kPartWideK ? 1 : kPartTilesPerSM) * kPartSMs;
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
  const int bmax = std::max(pl.b0, std::max(pl.b1, pl.b2));
  const bool tcur_smem = tags && scatter_smem_words(K, bmax, true, true) * sizeof(uint32_t) <= kMaxSmemScatter;
  const size_t sms = scatter_smem_words(K, bmax, tags, tcur_smem) * sizeof(uint32_t);
  auto count = tags ? part_count_kernel<true> : part_count_kernel<false>;
  ScatterFn scatter = tags ? scatter_fn<true>(pl.b0, pl.b1, pl.b2) : scatter_fn<false>(pl.b0, pl.b1, pl.b2);
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
  // a single tile without tag lists: the scatter CTA counts and scans itself
  const bool fused = !tags && pl.ntiles == 1;
  if (pl.ntiles > 0 && !fused) {
    count<<<(unsigned)pl.ntiles, kPThreads, smc, s>>>(labels, N, K, pl.tile, tilecnt, tags ? tl->tag_off : nullptr,
                                                      tagcnt, hdr);
    count_launch();
  }
  if (!fused) {
    part_colscan_kernel<int32_t><<<(K + 31) / 32, 1024, 0, s>>>(tilecnt, pl.ntiles, K, hist);
    part_offsets_kernel<<<1, 1024, 0, s>>>(hist, K, offsets);
    count_launch(2);
  }
  if (tags) {
    part_colscan_kernel<int64_t><<<(K + 31) / 32, 1024, 0, s>>>(tagcnt, pl.ntiles, K, tag_hist);
    part_offsets_kernel<<<1, 1024, 0, s>>>(tag_hist, K, tag_base);
    count_launch(2);
  }
  if (pl.ntiles > 0) {
    TagArgs ta{};
    if (tags) ta = TagArgs{tl->tag_off, tl->tags, tagcnt, tag_base, tl->tag_off_out, tl->tags_out, tcur_smem ? 1 : 0};
    scatter<<<(unsigned)pl.ntiles, kSThreads, sms, s>>>(labels, N, K, pl.tile, fused ? nullptr : tilecnt, offsets,
                                                        perm, ta, fused ? hist : nullptr, fused ? offsets : nullptr, hdr);
    count_launch();
    if (sorted_labels) {
      const int64_t per = (int64_t)kFillThreads * kFillSlots;
      part_fill_labels_kernel<<<(unsigned)((N + per - 1) / per), kFillThreads, 0, s>>>(offsets, K, N, sorted_labels);
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
