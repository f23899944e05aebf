// init.cu -- k-means++ seeding (Arthur & Vassilvitskii 2007) of the gater's
// centres.  The paper asks for "K-means clustering" of the features (Section 2)
// and names no initialisation; this is the stated reading:
//   candidates  all N rows, or m = min(N, 256 K) rows drawn with replacement:
//               candidate j = row floor(u_j N), u_j from splitmix64 output j
//               of (seed ^ kSubsampleStream);
//   round 0     candidate floor(u m), u from splitmix64 output 0 of seed;
//   round k     D^2 (fp64) = squared distance of every candidate to its
//               nearest chosen centre; the pick is the smallest candidate
//               whose running total of D^2 exceeds u * sum(D^2), u from
//               splitmix64 output k of seed; if the sum is 0, floor(u m).
// splitmix64 (Steele, Lea, Flood 2014) is counter-indexable: output j of the
// generator seeded with s is mix(s + (j + 1) * 0x9E3779B97F4A7C15).
// One launch of the distance kernel and one of the pick kernel per round.
#include "hme_common.cuh"

namespace hme {

namespace {

constexpr uint64_t kGolden = 0x9E3779B97F4A7C15ull;
constexpr uint64_t kSubsampleStream = 0xD1B54A32D192ED03ull;
constexpr int kCandPerBlock = 256;

__device__ __forceinline__ uint64_t splitmix64_at(uint64_t seed, uint64_t j) {
  uint64_t z = seed + (j + 1) * kGolden;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// floor(u * n) with u = (r >> 11) / 2^53, exactly: the high 64 bits of (r with its low 11 bits cleared) * n.
__device__ __forceinline__ uint64_t scaled_index(uint64_t r, uint64_t n) {
  return __umul64hi(r & ~0x7FFull, n);
}

__device__ __forceinline__ double unit53(uint64_t r) { return (double)(r >> 11) * (1.0 / 9007199254740992.0); }

template <int DT>
__device__ __forceinline__ float feat(const void *X, int64_t off) {
  if (DT == HME_BF16) return __bfloat162float(static_cast<const __nv_bfloat16 *>(X)[off]);
  return static_cast<const float *>(X)[off];
}

__global__ void kpp_rows_kernel(int32_t *rows, int64_t m, int64_t N, uint64_t seed, int sampled) {
  const int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= m) return;
  rows[j] = sampled ? (int32_t)scaled_index(splitmix64_at(seed ^ kSubsampleStream, (uint64_t)j), (uint64_t)N)
                    : (int32_t)j;
}

template <int DT>
__global__ void kpp_first_kernel(const void *X, int d, int64_t ldx, const int32_t *rows, int64_t m, uint64_t seed,
                                 float *C, Header *hdr) {
  const int64_t pick = (int64_t)scaled_index(splitmix64_at(seed, 0), (uint64_t)m);
  const int64_t row = rows[pick];
  for (int j = threadIdx.x; j < d; j += blockDim.x) C[j] = feat<DT>(X, row * ldx + j);
  if (threadIdx.x == 0) hdr->kpp_choice = (uint32_t)pick;
}

// D2[j] = min(D2[j], ||x_rows[j] - c||^2) in fp64 (first round: assignment);
// part[b] = sum of this block's D2 in candidate order.
template <int DT>
__global__ void __launch_bounds__(256) kpp_dist_kernel(const void *X, int d, int64_t ldx,
                                                       const int32_t *__restrict__ rows, int64_t m,
                                                       const float *__restrict__ c, double *D2, int first,
                                                       double *part) {
  __shared__ double vals[kCandPerBlock];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t b0 = (int64_t)blockIdx.x * kCandPerBlock;
  for (int q = warp; q < kCandPerBlock; q += 8) {
    const int64_t j = b0 + q;
    double v = 0.0;
    if (j < m) {
      const int64_t row = rows[j];
      double s = 0.0;
      for (int e = lane; e < d; e += 32) {
        const double t = (double)feat<DT>(X, row * ldx + e) - (double)c[e];
        s = fma(t, t, s);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
      v = first ? s : fmin(D2[j], s);
      if (lane == 0) D2[j] = v;
    }
    if (lane == 0) vals[q] = v;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int q = 0; q < kCandPerBlock; ++q) t += vals[q];
    part[blockIdx.x] = t;
  }
}

// Round k: draw u, walk the running total of D^2 (block partials, then the
// block's own candidates) to the first candidate whose running total > u * sum.
template <int DT>
__global__ void kpp_pick_kernel(const void *X, int d, int64_t ldx, const int32_t *rows, int64_t m,
                                const double *D2, const double *part, int64_t nb, uint64_t seed, int k, float *Ck,
                                Header *hdr) {
  __shared__ int64_t s_pick;
  if (threadIdx.x == 0) {
    double total = 0.0;
    for (int64_t b = 0; b < nb; ++b) total += part[b];
    const uint64_t r = splitmix64_at(seed, (uint64_t)k);
    int64_t pick = -1;
    if (total > 0.0) {
      const double thr = unit53(r) * total;
      double run = 0.0;
      int64_t blk = -1;
      for (int64_t b = 0; b < nb; ++b) {
        if (run + part[b] > thr) {
          blk = b;
          break;
        }
        run += part[b];
      }
      if (blk >= 0) {
        const int64_t j1 = min(m, (blk + 1) * (int64_t)kCandPerBlock);
        for (int64_t j = blk * kCandPerBlock; j < j1; ++j) {
          run += D2[j];
          if (run > thr) {
            pick = j;
            break;
          }
        }
      }
      if (pick < 0)  // rounding put the threshold past the last total: the last candidate with D^2 > 0
        for (int64_t j = m - 1; j >= 0; --j)
          if (D2[j] > 0.0) {
            pick = j;
            break;
          }
    }
    if (pick < 0) pick = (int64_t)scaled_index(r, (uint64_t)m);
    s_pick = pick;
    hdr->kpp_choice = (uint32_t)pick;
  }
  __syncthreads();
  const int64_t row = rows[s_pick];
  for (int j = threadIdx.x; j < d; j += blockDim.x) Ck[j] = feat<DT>(X, row * ldx + j);
}

__global__ void debug_wait_kernel(uint64_t limit_ns, Header *hdr) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(smem_u32(&bar), 1);
    fence_mbar_init();
    // Nothing ever arrives on this barrier: the wait must expire and report.
    mbar_wait_bounded(smem_u32(&bar), 0, limit_ns, hdr, 99);
  }
}

}  // namespace

int64_t kpp_candidates(int64_t N, int K, int method) {
  if (method == HME_INIT_KMEANSPP_SUBSAMPLE && N > 256 * (int64_t)K) return 256 * (int64_t)K;
  return N;
}

int64_t kpp_blocks(int64_t m) { return (m + kCandPerBlock - 1) / kCandPerBlock; }

cudaError_t launch_kmeanspp(const void *X, int64_t N, int d, int64_t ldx, int dtype, int K, uint64_t seed,
                            int64_t m, bool subsample, float *C_out, int32_t *rows, double *d2, double *part,
                            Header *hdr, cudaStream_t s) {
  const int sampled = subsample && m < N;
  kpp_rows_kernel<<<(unsigned)((m + 255) / 256), 256, 0, s>>>(rows, m, N, seed, sampled);
  const int64_t nb = kpp_blocks(m);
  if (dtype == HME_BF16)
    kpp_first_kernel<HME_BF16><<<1, 256, 0, s>>>(X, d, ldx, rows, m, seed, C_out, hdr);
  else
    kpp_first_kernel<HME_F32><<<1, 256, 0, s>>>(X, d, ldx, rows, m, seed, C_out, hdr);
  count_launch(2);
  for (int k = 1; k < K; ++k) {
    const float *cprev = C_out + (int64_t)(k - 1) * d;
    float *ck = C_out + (int64_t)k * d;
    if (dtype == HME_BF16) {
      kpp_dist_kernel<HME_BF16><<<(unsigned)nb, 256, 0, s>>>(X, d, ldx, rows, m, cprev, d2, k == 1, part);
      kpp_pick_kernel<HME_BF16><<<1, 256, 0, s>>>(X, d, ldx, rows, m, d2, part, nb, seed, k, ck, hdr);
    } else {
      kpp_dist_kernel<HME_F32><<<(unsigned)nb, 256, 0, s>>>(X, d, ldx, rows, m, cprev, d2, k == 1, part);
      kpp_pick_kernel<HME_F32><<<1, 256, 0, s>>>(X, d, ldx, rows, m, d2, part, nb, seed, k, ck, hdr);
    }
    count_launch(2);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return cudaGetLastError();
}

cudaError_t launch_debug_wait(uint64_t timeout_ns, Header *hdr, cudaStream_t s) {
  debug_wait_kernel<<<1, 32, 0, s>>>(timeout_ns, hdr);
  count_launch();
  return cudaGetLastError();
}

}  // namespace hme
