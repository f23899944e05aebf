// pca.cu -- principal components of the gater features (Section 4.2, "Model
// and training details": before the K-means, Z = T^{L-1}(X) is projected onto
// its first 256 principal directions).  Readings: centred about the column
// mean, covariance normalised by N, unwhitened projection, components in
// decreasing variance with the entry of largest magnitude positive.
//
// Fit:
//   pca_colsum      per-slab column sums of X (fp32 over 32 rows, fp64 across);
//   pca_mean        the slab sums added in slab order / N -> mu (fp64, fp32);
//   pca_split_t     y = x - mu (fp32) split into bf16 y = yh + yl + O(2^-16 |y|),
//                   written transposed in blocks of R rows (each block a d x R
//                   matrix, one row per feature), so that the covariance is a
//                   K-major contraction over the rows for the tensor cores;
//   pca_cov         tcgen05 (kind::f16, fp32 accumulate in TMEM): work units
//                   are (block of rows, 128 x 128 tile (i <= j) of the upper
//                   triangle); a unit accumulates yh.yh' + yh.yl' + yl.yh' in
//                   TMEM over kCovSub rows at a time (short fp32 sums), its
//                   epilogue adds each such sub-result into fp32 registers
//                   (round to nearest) while the MMAs of the next sub-range run
//                   in the other accumulator, and stores its fp32 partial tile
//                   once (a block has at most kCovFlush sub-ranges);
//   pca_cov_reduce  the partial tiles added in range order in fp64, / N: the
//                   covariance (fp64, both triangles) and A (fp32, order n = d
//                   rounded up to even, padding row and column zero);
//   Jacobi          cyclic two-sided block Jacobi on A (n = d rounded up to a
//                   multiple of 64; blocks of 32 indices paired by the circle
//                   method): per round, the 64 x 64 sub-problems of the block
//                   pairs are diagonalised in shared memory and their
//                   orthogonal factors applied to the rest of A and to V (the
//                   eigenvector estimate) as fp32 64 x 64 products, in place.
//                   Sweeps repeat until off(A) <= 2^-20 ||A||_F;
//   pca_rank        eigenvalues diag(A) ranked (decreasing, ties to the lower
//                   index), the padding slot excluded;
//   pca_components  the leading r columns of V, normalised, with the sign rule.
// Transform: hme_pca_transform runs the assign kernel that splits fp32 rows in
// the kernel, with the components as its centres, in projection mode.
#include <mutex>

#include "hme_common.cuh"

namespace hme {

namespace {

constexpr int kColThreads = 256;
constexpr int kColSlab = 2048;  // rows per column-sum block
constexpr int kCovThreads = 320;  // warp 0 TMA, warp 1 MMA, warps 2-9 epilogue (two per TMEM lane quarter)
constexpr int kCovHalf = kBM / 2;  // accumulator columns per epilogue warp
constexpr int kCovStages = 3;
constexpr uint32_t kCovOpBytes = kBM * kBK * 2;  // 128 rows x 64 bf16 = 16 KB
constexpr uint32_t kCovStageBytes = 4 * kCovOpBytes;  // A hi, A lo, B hi, B lo
constexpr uint32_t kCovTmemCols = 256;  // two 128-column accumulators
constexpr uint32_t kWhereCovProducer = 11, kWhereCovMma = 12, kWhereCovEpi = 13;

// ---------------------------------------------------------------------------
// mean and centred transposed split
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kColThreads) pca_colsum_kernel(const float *__restrict__ X, int64_t N, int d,
                                                                 int64_t ldx, double *__restrict__ part) {
  const int f = blockIdx.x * kColThreads + threadIdx.x;
  if (f >= d) return;
  const int64_t r0 = (int64_t)blockIdx.y * kColSlab;
  const int64_t r1 = N < r0 + kColSlab ? N : r0 + kColSlab;
  double acc = 0.0;
  for (int64_t i = r0; i < r1; i += 32) {
    const int64_t e = r1 < i + 32 ? r1 : i + 32;
    float s = 0.0f;
#pragma unroll 8
    for (int64_t k = i; k < e; ++k) s += __ldg(X + k * ldx + f);
    acc += (double)s;
  }
  part[(int64_t)blockIdx.y * d + f] = acc;
}

__global__ void pca_mean_kernel(const double *__restrict__ part, int64_t nslabs, int64_t N, int d,
                                double *__restrict__ mean64, float *__restrict__ mean32) {
  const int f = blockIdx.x * blockDim.x + threadIdx.x;
  if (f >= d) return;
  double s = 0.0;
  for (int64_t b = 0; b < nslabs; ++b) s += part[b * d + f];
  const double m = s / (double)N;
  mean64[f] = m;
  mean32[f] = (float)m;
}

__device__ __forceinline__ void split_bf16(float y, uint16_t &h, uint16_t &l) {
  const __nv_bfloat16 hb = __float2bfloat16_rn(y);
  const __nv_bfloat16 lb = __float2bfloat16_rn(y - __bfloat162float(hb));
  h = __bfloat16_as_ushort(hb);
  l = __bfloat16_as_ushort(lb);
}

// A block moves 64 rows x 64 features: loads coalesced along the features,
// stores coalesced along the rows (128 bytes per feature row) into block
// n / R of the transposed split.  Rows past N (the padding of the last block)
// are written as zeros.
constexpr int kTPad = 66;  // shared row pitch in 16-bit elements (33 words: few bank conflicts)
template <bool VEC>
__global__ void __launch_bounds__(256) pca_split_t_kernel(const float *__restrict__ X, int64_t N, int d, int64_t ldx,
                                                          const float *__restrict__ mu, int64_t R,
                                                          __nv_bfloat16 *__restrict__ yh,
                                                          __nv_bfloat16 *__restrict__ yl) {
  __shared__ __align__(16) uint16_t sh[64 * kTPad];
  __shared__ __align__(16) uint16_t sl[64 * kTPad];
  const int64_t n0 = (int64_t)blockIdx.x * 64;
  const int f0 = blockIdx.y * 64;
  const int t = threadIdx.x;
  const int c4 = (t & 15) * 4;
  float m[4];
#pragma unroll
  for (int e = 0; e < 4; ++e) m[e] = f0 + c4 + e < d ? __ldg(mu + f0 + c4 + e) : 0.0f;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int rr = (t >> 4) + 16 * k;
    const int64_t n = n0 + rr;
    float v[4] = {0.0f, 0.0f, 0.0f, 0.0f};
    if (n < N) {
      const float *src = X + n * ldx + f0 + c4;
      if (VEC && f0 + c4 + 3 < d) {
        const float4 q = __ldg(reinterpret_cast<const float4 *>(src));
        v[0] = q.x - m[0], v[1] = q.y - m[1], v[2] = q.z - m[2], v[3] = q.w - m[3];
      } else {
#pragma unroll
        for (int e = 0; e < 4; ++e)
          if (f0 + c4 + e < d) v[e] = __ldg(src + e) - m[e];
      }
    }
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      uint16_t h, l;
      split_bf16(v[e], h, l);
      sh[(c4 + e) * kTPad + rr] = h;
      sl[(c4 + e) * kTPad + rr] = l;
    }
  }
  __syncthreads();
#pragma unroll
  // the 64 rows lie in one block c of R rows (R is a multiple of 64)
  const int64_t c = n0 / R, x0 = n0 - c * R;
  for (int k = 0; k < 2; ++k) {
    const int idx = t + 256 * k;  // 64 features x 8 chunks of 8 rows
    const int ff = idx >> 3, ch = idx & 7;
    const int f = f0 + ff;
    if (f < d) {
      const uint32_t *ph = reinterpret_cast<const uint32_t *>(sh + ff * kTPad + ch * 8);
      const uint32_t *pl = reinterpret_cast<const uint32_t *>(sl + ff * kTPad + ch * 8);
      const int64_t o = (c * d + f) * R + x0 + ch * 8;
      *reinterpret_cast<uint4 *>(yh + o) = make_uint4(ph[0], ph[1], ph[2], ph[3]);
      *reinterpret_cast<uint4 *>(yl + o) = make_uint4(pl[0], pl[1], pl[2], pl[3]);
    }
  }
}

// ---------------------------------------------------------------------------
// covariance: tcgen05 over chunks of rows, upper-triangle tiles
// ---------------------------------------------------------------------------
struct CovParams {
  int64_t N;
  int64_t R;       // rows per unit range (multiple of kCovSub)
  int mi;          // 128-feature tiles along d
  int ntiles;      // mi (mi + 1) / 2
  int64_t nunits;  // ranges x tiles
  float *part;     // [nunits][128][128]
  Header *hdr;
  uint64_t limit_ns;
};
constexpr int kSubKb = (int)(kCovSub / kBK);  // k-blocks per TMEM accumulation

// tile t of the upper triangle, enumerated row by row: (i, j), i <= j
__device__ __forceinline__ void cov_tile(int t, int mi, int &i, int &j) {
  int a = 0;
  while (t >= mi - a) {
    t -= mi - a;
    ++a;
  }
  i = a;
  j = a + t;
}

__global__ void __launch_bounds__(kCovThreads, 1)
    pca_cov_kernel(const __grid_constant__ CUtensorMap tmH, const __grid_constant__ CUtensorMap tmL,
                   const CovParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_addr = smem_u32(smem_raw);
  const uint32_t base = (raw_addr + 1023u) & ~1023u;
  uint8_t *smem = smem_raw + (base - raw_addr);
  constexpr int S = kCovStages;
  const uint32_t ring = base;
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + S * kCovStageBytes);
  uint64_t *empty = full + S;
  uint64_t *tfull = empty + S;
  uint64_t *tempty = tfull + 2;
  uint64_t *drain = tempty + 2;
  uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(drain + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_u32(&tfull[a]), 1);
      mbar_init(smem_u32(&tempty[a]), 8);
    }
    mbar_init(smem_u32(drain), 1);
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tensormap(&tmH);
    prefetch_tensormap(&tmL);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_holder), kCovTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;

  auto kblocks = [&](int64_t c) -> int {
    const int64_t rows = p.N - c * p.R < p.R ? p.N - c * p.R : p.R;
    return (int)((rows + kBK - 1) / kBK);
  };

  if (warp == 0) {
    if (lane == 0) {
      const uint64_t pol = l2_policy_evict_last();  // a chunk is read by every tile of the triangle
      uint32_t it = 0;
      bool ok = true;
      for (int64_t u = blockIdx.x; u < p.nunits && ok; u += gridDim.x) {
        const int64_t c = u / p.ntiles;
        int i, j;
        cov_tile((int)(u - c * p.ntiles), p.mi, i, j);
        const int nkb = kblocks(c);
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const int s = it % S;
          if (!mbar_wait_bounded(smem_u32(&empty[s]), ((it / S) & 1u) ^ 1u, p.limit_ns, p.hdr, kWhereCovProducer)) {
            ok = false;
            break;
          }
          const uint32_t fb = smem_u32(&full[s]);
          mbar_arrive_expect_tx(fb, kCovStageBytes);
          const uint32_t st = ring + (uint32_t)s * kCovStageBytes;
          const int32_t x = kb * kBK, z = (int32_t)c;  // column within block c
          tma_load_3d(st, &tmH, fb, x, i * kBM, z, pol);
          tma_load_3d(st + kCovOpBytes, &tmL, fb, x, i * kBM, z, pol);
          tma_load_3d(st + 2 * kCovOpBytes, &tmH, fb, x, j * kBM, z, pol);
          tma_load_3d(st + 3 * kCovOpBytes, &tmL, fb, x, j * kBM, z, pol);
        }
      }
      if (!ok) {  // every copy issued must land before the CTA ends
        for (uint32_t q = (it > (uint32_t)S ? it - S : 0); q < it; ++q)
          mbar_wait_bounded(smem_u32(&full[q % S]), (q / S) & 1u, 200000000ull, p.hdr, kWhereCovProducer);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(kBM, kBM);
      uint32_t it = 0, acc_it = 0;
      bool ok = true;
      for (int64_t u = blockIdx.x; u < p.nunits && ok; u += gridDim.x) {
        const int nkb = kblocks(u / p.ntiles);
        for (int kb0 = 0; kb0 < nkb && ok; kb0 += kSubKb, ++acc_it) {
          const uint32_t a = acc_it & 1u;
          if (!mbar_wait_bounded(smem_u32(&tempty[a]), ((acc_it >> 1) & 1u) ^ 1u, p.limit_ns, p.hdr, kWhereCovMma)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t dt = tmem_base + a * (uint32_t)kBM;
          const int kb1 = nkb < kb0 + kSubKb ? nkb : kb0 + kSubKb;
          for (int kb = kb0; kb < kb1; ++kb, ++it) {
            const int s = it % S;
            if (!mbar_wait_bounded(smem_u32(&full[s]), (it / S) & 1u, p.limit_ns, p.hdr, kWhereCovMma)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t st = ring + (uint32_t)s * kCovStageBytes;
#pragma unroll
            for (int k = 0; k < kBK / 16; ++k) {
              const uint64_t ah = smem_desc_sw128(st + k * 32);
              const uint64_t al = smem_desc_sw128(st + kCovOpBytes + k * 32);
              const uint64_t bh = smem_desc_sw128(st + 2 * kCovOpBytes + k * 32);
              const uint64_t bl = smem_desc_sw128(st + 3 * kCovOpBytes + k * 32);
              tc_mma_bf16(dt, ah, bh, idesc, (kb > kb0 || k > 0) ? 1u : 0u);
              tc_mma_bf16(dt, ah, bl, idesc, 1u);  // yh . yl'
              tc_mma_bf16(dt, al, bh, idesc, 1u);  // yl . yh'
            }
            tc_commit(smem_u32(&empty[s]));
          }
          if (ok) tc_commit(smem_u32(&tfull[a]));
        }
      }
      if (!ok) {
        tc_commit(smem_u32(drain));
        mbar_wait_bounded(smem_u32(drain), 0, 200000000ull, p.hdr, kWhereCovMma);
      }
    }
  } else {
    // epilogue: accumulator row (TMEM lane), half of its columns -> the partial tile
    const int q = warp & 3;
    const int row = q * 32 + lane;
    const int col0 = ((warp - 2) >> 2) * kCovHalf;
    // Each sub-range sum (one TMEM accumulation, at most kCovFlush per unit)
    // is added into fp32 registers (round to nearest); the unit's partial
    // tile row is stored once at its end.
    uint32_t acc_it = 0;
    bool ok = true;
    float acc[kCovHalf];
    for (int64_t u = blockIdx.x; u < p.nunits && ok; u += gridDim.x) {
      const int nkb = kblocks(u / p.ntiles);
      float *dst = p.part + u * (int64_t)(kBM * kBM) + (int64_t)row * kBM + col0;
#pragma unroll
      for (int c = 0; c < kCovHalf; ++c) acc[c] = 0.0f;
      for (int kb0 = 0; kb0 < nkb; kb0 += kSubKb, ++acc_it) {
        const uint32_t a = acc_it & 1u;
        if (!mbar_wait_bounded(smem_u32(&tfull[a]), (acc_it >> 1) & 1u, p.limit_ns, p.hdr, kWhereCovEpi)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t taddr = tmem_base + a * (uint32_t)kBM + (uint32_t)col0 + ((uint32_t)(q * 32) << 16);
        uint32_t r0[16], r1[16];
#pragma unroll
        for (int c = 0; c < kCovHalf; c += 32) {
          tmem_ld16(taddr + (uint32_t)c, r0);
          tmem_ld16(taddr + (uint32_t)(c + 16), r1);
          tmem_ld_wait(r0);
          tmem_ld_wait(r1);
#pragma unroll
          for (int e = 0; e < 16; ++e) {
            acc[c + e] += __uint_as_float(r0[e]);
            acc[c + 16 + e] += __uint_as_float(r1[e]);
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&tempty[a]));
      }
      if (!ok) break;
#pragma unroll
      for (int c = 0; c < kCovHalf; c += 4)
        *reinterpret_cast<float4 *>(dst + c) = make_float4(acc[c], acc[c + 1], acc[c + 2], acc[c + 3]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kCovTmemCols);
  }
}

// cov[a][b] = cov[b][a] = (sum over chunks of the partial entries, fp64, in
// chunk order) / N for a <= b; A (order n) gets the same values in fp32.
__global__ void __launch_bounds__(256) pca_cov_reduce_kernel(const float *__restrict__ part, int64_t nchunks,
                                                             int ntiles, int mi, int d, int n, int64_t N,
                                                             double *__restrict__ cov, float *__restrict__ A) {
  if (blockIdx.x < blockIdx.y) return;  // 32 x 32 blocks wholly below the diagonal
  const int b = blockIdx.x * 32 + (threadIdx.x & 31);
  const int a0 = blockIdx.y * 32;
  for (int aa = threadIdx.x >> 5; aa < 32; aa += 8) {
    const int a = a0 + aa;
    if (a >= d || b >= d || b < a) continue;
    const int i = a >> 7, j = b >> 7;
    const int t = i * mi - i * (i - 1) / 2 + (j - i);
    const int64_t off = (int64_t)t * (kBM * kBM) + (int64_t)(a & 127) * kBM + (b & 127);
    const int64_t stride = (int64_t)ntiles * (kBM * kBM);
    double s = 0.0;
    for (int64_t c = 0; c < nchunks; ++c) s += (double)part[c * stride + off];
    const double v = s / (double)N;
    if (cov) {
      cov[(int64_t)a * d + b] = v;
      cov[(int64_t)b * d + a] = v;
    }
    A[(int64_t)a * n + b] = (float)v;
    A[(int64_t)b * n + a] = (float)v;
  }
}

// ---------------------------------------------------------------------------
// Jacobi
// ---------------------------------------------------------------------------
// Circle-method ordering on fixed positions (no data movement): with
// m = n - 1, round t in [0, m) pairs index 0 with 1 + t (pair 0) and, for
// k = 1 .. n/2 - 1, p_k = 1 + (t + k) mod m with q_k = 1 + (t - k) mod m; over
// m rounds every two indices meet once.  Consecutive pairs k touch ascending
// (p) and descending (q) consecutive indices, so a warp's accesses to a row
// stay contiguous.
__device__ __forceinline__ int jac_p(int k, int t, int m) {
  if (k == 0) return 0;
  const int x = t + k;
  return 1 + (x >= m ? x - m : x);
}
__device__ __forceinline__ int jac_q(int k, int t, int m) {
  if (k == 0) return 1 + t;
  const int x = t - k;
  return 1 + (x < 0 ? x + m : x);
}
// The rotation of one pair (Rutishauser's form): t = tan(phi) is the smaller
// root of t^2 + 2 theta t - 1 = 0, theta = (a_qq - a_pp) / (2 a_pq), which
// zeroes a_pq; the update of a pair of entries (u, v) of rows (or columns) p
// and q is u - s (v + tau u), v + s (u - tau v) with s = sin(phi), tau =
// tan(phi / 2), which keeps the norm of (u, v) to second order in s even when
// cos(phi) rounds to 1.  Entries with |a_pq| <= 2^-23 sqrt(|a_pp| |a_qq|) are
// left alone.  Returns (s, tau, dp, dq), dp and dq the new diagonal entries.
// Each rotation is computed once per round, by one thread.
__device__ float4 jac_rot4(float app, float aqq, float apq) {
  float4 r = make_float4(0.0f, 0.0f, app, aqq);
  if (apq != 0.0f && fabsf(apq) > 0x1p-23f * sqrtf(fabsf(app)) * sqrtf(fabsf(aqq))) {
    const float theta = (aqq - app) / (2.0f * apq);
    const float at = fabsf(theta);
    float t = at > 0x1p20f ? 0.5f / at : 1.0f / (at + sqrtf(at * at + 1.0f));
    t = copysignf(t, theta);
    const float c = 1.0f / sqrtf(t * t + 1.0f);
    r.x = t * c;
    r.y = r.x / (1.0f + c);
    r.z = app - t * apq;
    r.w = aqq + t * apq;
  }
  return r;
}

// Blocked Jacobi.  The order n is a multiple of 2 kJB; the n / kJB blocks of
// kJB indices are paired by the same circle method (round t of nb - 1, pair P
// = blocks (jac_p(P, t, nb - 1), jac_q(P, t, nb - 1))).  A round:
//   bj_sub_kernel    one CTA per block pair: one cyclic Jacobi sweep (the
//                    scalar rotations above, 63 rounds) on the 64 x 64
//                    sub-matrix S of A on the pair's indices, in shared memory
//                    (more inner sweeps per round saved at most one outer sweep
//                    in a prototype, and cost a full sweep each); its orthogonal
//                    factor Q (S <- Q^T S Q, a product of rotations close to the
//                    identity, never a permutation: eigenvectors sorted by
//                    eigenvalue stalled the outer iteration in the prototype)
//                    goes to Qbuf and S back into A;
//   bj_apply_kernel  A_PR <- Q_P^T A_PR Q_R for every other 64 x 64 tile of A
//                    on pairs (P, R), and V_kR <- V_kR Q_R for every 64-row
//                    slice of V: two fp32 64 x 64 x 64 products per tile in
//                    shared memory, each tile read and written in place by
//                    one CTA.
// A sweep (nb - 1 rounds) meets every pair of blocks once, so every pair of
// indices, as the scalar method does; it passes over A and V 2 (nb - 1) times
// instead of n - 1.
constexpr int kJB = 32;        // indices per block
constexpr int kJS = 2 * kJB;   // order of a sub-problem
constexpr int kJSP = kJS + 1;  // shared row pitch of the sub-problem kernel
constexpr int kApT = 68;       // shared row pitch of the apply kernel (16-byte rows)

__device__ __forceinline__ int bj_index(int i, int I, int J) { return i < kJB ? I * kJB + i : J * kJB + (i - kJB); }

// One thread per 2 x 2 block of S and two column pairs of Q per inner round;
// the inner rounds' pairs come from a table.  Each inner round: the 32
// rotations (one warp), a barrier, the updates of S and Q, a barrier.
constexpr int kSubThreads = 1024;
__global__ void __launch_bounds__(kSubThreads) bj_sub_kernel(float *__restrict__ A, int n, int t,
                                                             float *__restrict__ Qbuf) {
  __shared__ float S[kJS * kJSP];
  __shared__ float Q[kJS * kJSP];
  __shared__ float4 rot[kJB];
  __shared__ uint8_t pq[kJS - 1][kJB][2];
  const int nbm = n / kJB - 1;
  const int P = blockIdx.x;
  const int I = jac_p(P, t, nbm), J = jac_q(P, t, nbm);
  for (int e = threadIdx.x; e < kJS * kJS; e += blockDim.x) {
    const int i = e / kJS, j = e - i * kJS;
    S[i * kJSP + j] = A[(int64_t)bj_index(i, I, J) * n + bj_index(j, I, J)];
    Q[i * kJSP + j] = i == j ? 1.0f : 0.0f;
  }
  for (int e = threadIdx.x; e < (kJS - 1) * kJB; e += blockDim.x) {
    const int r = e / kJB, k = e - r * kJB;
    pq[r][k][0] = (uint8_t)jac_p(k, r, kJS - 1);
    pq[r][k][1] = (uint8_t)jac_q(k, r, kJS - 1);
  }
  __syncthreads();
  const int K = threadIdx.x / kJB, L = threadIdx.x % kJB;  // this thread's 2 x 2 block of S
  const int qi = threadIdx.x / (kJB / 2), qL0 = (threadIdx.x % (kJB / 2)) * 2;  // Q row, two column pairs
  for (int r = 0; r < kJS - 1; ++r) {
    if (threadIdx.x < kJB) {
      const int p = pq[r][threadIdx.x][0], q = pq[r][threadIdx.x][1];
      rot[threadIdx.x] = jac_rot4(S[p * kJSP + p], S[q * kJSP + q], S[p * kJSP + q]);
    }
    __syncthreads();
    {
      const int pK = pq[r][K][0], qK = pq[r][K][1], pL = pq[r][L][0], qL = pq[r][L][1];
      const float4 rk = rot[K];
      float *sp = S + pK * kJSP, *sq = S + qK * kJSP;
      if (K == L) {
        sp[pL] = rk.z;
        sq[qL] = rk.w;
        sp[qL] = 0.0f;
        sq[pL] = 0.0f;
      } else {
        const float4 rl = rot[L];
        const float a00 = sp[pL], a01 = sp[qL], a10 = sq[pL], a11 = sq[qL];
        const float s1 = rk.x, t1 = rk.y, s2 = rl.x, t2 = rl.y;
        const float m00 = a00 - s1 * (a10 + t1 * a00), m10 = a10 + s1 * (a00 - t1 * a10);
        const float m01 = a01 - s1 * (a11 + t1 * a01), m11 = a11 + s1 * (a01 - t1 * a11);
        sp[pL] = m00 - s2 * (m01 + t2 * m00);
        sp[qL] = m01 + s2 * (m00 - t2 * m01);
        sq[pL] = m10 - s2 * (m11 + t2 * m10);
        sq[qL] = m11 + s2 * (m10 - t2 * m11);
      }
    }
#pragma unroll
    for (int c = 0; c < 2; ++c) {  // Q <- Q J on row qi, column pairs qL0, qL0 + 1
      const int Lq = qL0 + c;
      const int pL = pq[r][Lq][0], qL = pq[r][Lq][1];
      const float4 rl = rot[Lq];
      float *qrow = Q + qi * kJSP;
      const float v0 = qrow[pL], v1 = qrow[qL];
      qrow[pL] = v0 - rl.x * (v1 + rl.y * v0);
      qrow[qL] = v1 + rl.x * (v0 - rl.y * v1);
    }
    __syncthreads();
  }
  float *qo = Qbuf + (int64_t)P * kJS * kJS;
  for (int e = threadIdx.x; e < kJS * kJS; e += blockDim.x) {
    const int i = e / kJS, j = e - i * kJS;
    qo[e] = Q[i * kJSP + j];
    A[(int64_t)bj_index(i, I, J) * n + bj_index(j, I, J)] = S[i * kJSP + j];
  }
}

// 64 x 64 x 64 product in shared memory: out[i][j] = sum_k L[k][i] R[k][j]
// (the left operand transposed), pitch kApT; thread (ty, tx) of 16 x 16 makes
// rows 4 ty .. 4 ty + 3 and columns 4 tx .. 4 tx + 3.
__device__ __forceinline__ void bj_mm_tn(const float *Lm, const float *Rm, float (&o)[4][4], int ty, int tx) {
#pragma unroll
  for (int a = 0; a < 4; ++a)
#pragma unroll
    for (int b = 0; b < 4; ++b) o[a][b] = 0.0f;
#pragma unroll 8
  for (int k = 0; k < kJS; ++k) {
    const float4 l = *reinterpret_cast<const float4 *>(Lm + k * kApT + 4 * ty);
    const float4 rr = *reinterpret_cast<const float4 *>(Rm + k * kApT + 4 * tx);
    const float lv[4] = {l.x, l.y, l.z, l.w}, rv[4] = {rr.x, rr.y, rr.z, rr.w};
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
      for (int b = 0; b < 4; ++b) o[a][b] = fmaf(lv[a], rv[b], o[a][b]);
  }
}

// Tiles [0, np^2 - np): (P, R), P != R, of A; then (n / 64) x np slices of V.
__global__ void __launch_bounds__(256) bj_apply_kernel(float *__restrict__ A, float *__restrict__ V, int n, int t,
                                                       const float *__restrict__ Qbuf) {
  extern __shared__ float4 bj_smem[];
  float *T = reinterpret_cast<float *>(bj_smem);  // the tile, then the intermediate product (transposed)
  float *QL = T + kJS * kApT;
  float *QR = QL + kJS * kApT;
  const int nb = n / kJB, nbm = nb - 1, np = nb / 2;
  const int ntile_a = np * np - np;
  const int ntiles = ntile_a + (n / kJS) * np;
  const int ty = threadIdx.x >> 4, tx = threadIdx.x & 15;
  for (int tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
    const bool isA = tile < ntile_a;
    int P = 0, R, row0 = 0;
    if (isA) {
      P = tile / (np - 1);
      R = tile - P * (np - 1);
      if (R >= P) ++R;  // skip the diagonal tile
    } else {
      const int v = tile - ntile_a;
      row0 = (v / np) * kJS;
      R = v - (v / np) * np;
    }
    const int IR = jac_p(R, t, nbm), JR = jac_q(R, t, nbm);
    const int IP = isA ? jac_p(P, t, nbm) : 0, JP = isA ? jac_q(P, t, nbm) : 0;
    float *M = isA ? A : V;
    __syncthreads();  // the previous tile's buffers are free
    // 16-byte loads: a tile row is two runs of 32 floats (blocks IR and JR)
    for (int e = threadIdx.x; e < kJS * kJS / 4; e += blockDim.x) {
      const int i = e / (kJS / 4), j = (e - i * (kJS / 4)) * 4;
      const int64_t gi = isA ? bj_index(i, IP, JP) : row0 + i;
      *reinterpret_cast<float4 *>(T + i * kApT + j) =
          __ldg(reinterpret_cast<const float4 *>(M + gi * n + bj_index(j, IR, JR)));
      *reinterpret_cast<float4 *>(QR + i * kApT + j) =
          __ldg(reinterpret_cast<const float4 *>(Qbuf + (int64_t)R * kJS * kJS + i * kJS + j));
      if (isA)
        *reinterpret_cast<float4 *>(QL + i * kApT + j) =
            __ldg(reinterpret_cast<const float4 *>(Qbuf + (int64_t)P * kJS * kJS + i * kJS + j));
    }
    __syncthreads();
    float o[4][4];
    if (isA) {
      bj_mm_tn(QL, T, o, ty, tx);  // U = Q_P^T T
      __syncthreads();             // T is overwritten by U^T
#pragma unroll
      for (int b = 0; b < 4; ++b)
        *reinterpret_cast<float4 *>(T + (4 * tx + b) * kApT + 4 * ty) = make_float4(o[0][b], o[1][b], o[2][b], o[3][b]);
      __syncthreads();
    } else {
      // V: T' = T Q_R, i.e. the left operand is T itself: store it transposed
      float tt[4][4];
#pragma unroll
      for (int a = 0; a < 4; ++a) {
        const float4 v = *reinterpret_cast<const float4 *>(T + (4 * ty + a) * kApT + 4 * tx);
        tt[a][0] = v.x, tt[a][1] = v.y, tt[a][2] = v.z, tt[a][3] = v.w;
      }
      __syncthreads();
#pragma unroll
      for (int b = 0; b < 4; ++b)
        *reinterpret_cast<float4 *>(T + (4 * tx + b) * kApT + 4 * ty) =
            make_float4(tt[0][b], tt[1][b], tt[2][b], tt[3][b]);
      __syncthreads();
    }
    bj_mm_tn(T, QR, o, ty, tx);  // (U or T) Q_R with the left operand stored transposed
#pragma unroll
    for (int a = 0; a < 4; ++a) {  // columns 4 tx .. 4 tx + 3 lie in one block run: a 16-byte store
      const int i = 4 * ty + a;
      const int64_t gi = isA ? bj_index(i, IP, JP) : row0 + i;
      *reinterpret_cast<float4 *>(M + gi * n + bj_index(4 * tx, IR, JR)) = make_float4(o[a][0], o[a][1], o[a][2], o[a][3]);
    }
  }
}

__global__ void pca_identity_kernel(float *V, int n) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i < (int64_t)n * n) V[i] = (i / n == i % n) ? 1.0f : 0.0f;
}

// acc[0] += sum of squared off-diagonal entries, acc[1] += sum of squared
// diagonal entries (fp64).
__global__ void __launch_bounds__(256) jacobi_offnorm_kernel(const float *__restrict__ A, int n, double *acc) {
  double off = 0.0, dia = 0.0;
  const int64_t total = (int64_t)n * n;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const double v = (double)A[i];
    if (i / n == i % n)
      dia += v * v;
    else
      off += v * v;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    off += __shfl_xor_sync(0xffffffffu, off, o);
    dia += __shfl_xor_sync(0xffffffffu, dia, o);
  }
  __shared__ double so[8], sd[8];
  if ((threadIdx.x & 31) == 0) {
    so[threadIdx.x >> 5] = off;
    sd[threadIdx.x >> 5] = dia;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    double a = 0.0, b = 0.0;
    for (int w = 0; w < 8; ++w) a += so[w], b += sd[w];
    atomicAdd(acc, a);
    atomicAdd(acc + 1, b);
  }
}

// One block: rank of every eigenvalue among the d real ones (decreasing, ties
// to the lower index); the r leading ones go to order[] and variances[].
__global__ void __launch_bounds__(1024) pca_rank_kernel(const float *__restrict__ A, int n, int d, int r,
                                                        int32_t *__restrict__ order, float *__restrict__ variances) {
  extern __shared__ float lam[];
  for (int j = threadIdx.x; j < d; j += blockDim.x) lam[j] = A[(int64_t)j * n + j];
  __syncthreads();
  for (int j = threadIdx.x; j < d; j += blockDim.x) {
    const float v = lam[j];
    int rank = 0;
    for (int i = 0; i < d; ++i) rank += (lam[i] > v || (lam[i] == v && i < j)) ? 1 : 0;
    if (rank < r) {
      order[rank] = j;
      if (variances) variances[rank] = v;
    }
  }
}

// Block k: column order[k] of V, normalised (fp64 norm), sign so that the
// entry of largest magnitude (lowest index among equals) is positive.
__global__ void __launch_bounds__(256) pca_components_kernel(const float *__restrict__ V, int n, int d,
                                                             const int32_t *__restrict__ order,
                                                             float *__restrict__ W) {
  const int k = blockIdx.x;
  const int j = order[k];
  double ss = 0.0;
  unsigned long long best = 0;  // |v| bits << 32 | (~index): max = largest magnitude, then lowest index
  for (int m = threadIdx.x; m < d; m += blockDim.x) {
    const float v = V[(int64_t)m * n + j];
    ss += (double)v * (double)v;
    const unsigned long long key =
        ((unsigned long long)__float_as_uint(fabsf(v)) << 32) | (unsigned long long)(0xFFFFFFFFu - (uint32_t)m);
    best = key > best ? key : best;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    ss += __shfl_xor_sync(0xffffffffu, ss, o);
    const unsigned long long ob = __shfl_xor_sync(0xffffffffu, best, o);
    best = ob > best ? ob : best;
  }
  __shared__ double sss[8];
  __shared__ unsigned long long sb[8];
  __shared__ float scale;
  if ((threadIdx.x & 31) == 0) {
    sss[threadIdx.x >> 5] = ss;
    sb[threadIdx.x >> 5] = best;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    unsigned long long bb = 0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) {
      t += sss[w];
      bb = sb[w] > bb ? sb[w] : bb;
    }
    const int mbest = (int)(0xFFFFFFFFu - (uint32_t)(bb & 0xFFFFFFFFull));
    const float vb = V[(int64_t)mbest * n + j];
    const double inv = t > 0.0 ? 1.0 / sqrt(t) : 1.0;
    scale = (float)(vb < 0.0f ? -inv : inv);
  }
  __syncthreads();
  const float sc = scale;
  for (int m = threadIdx.x; m < d; m += blockDim.x) W[(int64_t)k * d + m] = V[(int64_t)m * n + j] * sc;
}

// zoff[j] = mu . w_j (fp64 sum, stored fp32) for j < r, 0 for r <= j < Kp.
__global__ void __launch_bounds__(256) pca_zoff_kernel(const float *__restrict__ mu, const float *__restrict__ W,
                                                       int d, int r, float *__restrict__ zoff) {
  const int j = blockIdx.x;
  double s = 0.0;
  if (j < r)
    for (int m = threadIdx.x; m < d; m += blockDim.x) s += (double)mu[m] * (double)W[(int64_t)j * d + m];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  __shared__ double ps[8];
  if ((threadIdx.x & 31) == 0) ps[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int w = 0; w < 8; ++w) t += ps[w];
    zoff[j] = (float)t;
  }
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// bf16 blocks of rows x cols (contiguous, row stride cols), nblk of them one
// after another; box = box_rows x 64 columns x 1 block, 128-byte swizzle.
int make_bf16_map_blocked(CUtensorMap *m, const void *ptr, uint64_t nblk, uint64_t rows, uint64_t cols,
                          uint32_t box_rows) {
  static EncodeTiledFn enc = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      enc = reinterpret_cast<EncodeTiledFn>(f);
  });
  if (!enc) return fail(HME_ECUDA, "cuTensorMapEncodeTiled is not available from the driver");
  cuuint64_t dims[3] = {cols, rows, nblk};
  cuuint64_t strides[2] = {cols * 2, rows * cols * 2};
  cuuint32_t box[3] = {(cuuint32_t)kBK, box_rows, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(ptr), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS)
    return fail(HME_ECUDA, "cuTensorMapEncodeTiled failed (%d) for %llu blocks of %llu x %llu", (int)r,
                (unsigned long long)nblk, (unsigned long long)rows, (unsigned long long)cols);
  return HME_OK;
}

}  // namespace

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
PcaGeom pca_geom(int64_t N, int d, int r) {
  PcaGeom g;
  g.N = N;
  g.d = d;
  g.r = r;
  g.n = (d + 63) / 64 * 64;

  g.mi = (d + kBM - 1) / kBM;
  g.ntiles = g.mi * (g.mi + 1) / 2;
  // Row ranges (= blocks of the transposed split) of at most kCovFlush
  // sub-ranges, and about 8 units per SM over all tiles (152 SMs assumed for
  // the sizing only).  A block is a contiguous d x R bf16 matrix: a k-block of
  // 64 rows then spans d x 2R bytes (32 MB at d = 2048), where a single d x N
  // matrix would put its 128-byte rows N x 2 bytes apart (2 MB at N = 10^6,
  // every row on its own page).
  int64_t ranges = (8 * 152 + g.ntiles - 1) / g.ntiles;
  const int64_t subs = (N + kCovSub - 1) / kCovSub;
  if (ranges > subs) ranges = subs > 0 ? subs : 1;
  int64_t per = (subs + ranges - 1) / ranges;
  if (per > kCovFlush) per = kCovFlush;
  g.R = per * kCovSub;
  g.nchunks = (N + g.R - 1) / g.R;
  g.ldn = g.nchunks * g.R;
  g.nslabs = (N + kColSlab - 1) / kColSlab;
  return g;
}

cudaError_t launch_pca_mean(const float *X, const PcaGeom &g, int64_t ldx, double *slab_sums, double *mean64,
                            float *mean32, cudaStream_t s) {
  const dim3 grid((unsigned)((g.d + kColThreads - 1) / kColThreads), (unsigned)g.nslabs);
  pca_colsum_kernel<<<grid, kColThreads, 0, s>>>(X, g.N, g.d, ldx, slab_sums);
  pca_mean_kernel<<<(g.d + 255) / 256, 256, 0, s>>>(slab_sums, g.nslabs, g.N, g.d, mean64, mean32);
  count_launch(2);
  return cudaGetLastError();
}

int launch_pca_cov(const float *X, const PcaGeom &g, int64_t ldx, const float *mean32, __nv_bfloat16 *yh,
                   __nv_bfloat16 *yl, float *part, double *cov, float *A, Header *hdr, cudaStream_t s) {
  const bool vec = (reinterpret_cast<uintptr_t>(X) & 15u) == 0 && ldx % 4 == 0;
  const dim3 tg((unsigned)(g.ldn / 64), (unsigned)((g.d + 63) / 64));  // every row of every block, padding included
  if (vec)
    pca_split_t_kernel<true><<<tg, 256, 0, s>>>(X, g.N, g.d, ldx, mean32, g.R, yh, yl);
  else
    pca_split_t_kernel<false><<<tg, 256, 0, s>>>(X, g.N, g.d, ldx, mean32, g.R, yh, yl);
  count_launch();
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "pca: split");
  CUtensorMap mH, mL;
  int rc;
  if ((rc = make_bf16_map_blocked(&mH, yh, (uint64_t)g.nchunks, (uint64_t)g.d, (uint64_t)g.R, kBM)) != HME_OK)
    return rc;
  if ((rc = make_bf16_map_blocked(&mL, yl, (uint64_t)g.nchunks, (uint64_t)g.d, (uint64_t)g.R, kBM)) != HME_OK)
    return rc;
  CovParams p;
  p.N = g.N;
  p.R = g.R;
  p.mi = g.mi;
  p.ntiles = g.ntiles;
  p.nunits = g.nchunks * g.ntiles;
  p.part = part;
  p.hdr = hdr;
  p.limit_ns = wait_limit_ns();
  const size_t smem = 1024 + (size_t)kCovStages * kCovStageBytes + 256;
  e = cudaFuncSetAttribute(pca_cov_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return cuda_fail(e, "pca: covariance smem");
  int grid = num_sms();
  if (grid > p.nunits) grid = (int)p.nunits;
  pca_cov_kernel<<<grid, kCovThreads, smem, s>>>(mH, mL, p);
  count_launch();
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "pca: covariance kernel launch");
  e = cudaMemsetAsync(A, 0, (size_t)g.n * g.n * sizeof(float), s);
  if (e != cudaSuccess) return cuda_fail(e, "pca: clear A");
  const dim3 rg((unsigned)((g.d + 31) / 32), (unsigned)((g.d + 31) / 32));
  pca_cov_reduce_kernel<<<rg, 256, 0, s>>>(part, g.nchunks, g.ntiles, g.mi, g.d, g.n, g.N, cov, A);
  count_launch();
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "pca: reduce");
  return HME_OK;
}

int run_pca_jacobi(const PcaGeom &g, float *A0, float *V0, float *Qbuf, double *acc, int32_t *order, float *W,
                   float *variances, int *sweeps_out, cudaStream_t s) {
  const int n = g.n;
  const int nb = n / kJB, np = nb / 2;
  pca_identity_kernel<<<(unsigned)(((int64_t)n * n + 255) / 256), 256, 0, s>>>(V0, n);
  count_launch();
  const size_t ap_smem = (size_t)3 * kJS * kApT * sizeof(float);
  cudaError_t ea = cudaFuncSetAttribute(bj_apply_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)ap_smem);
  if (ea != cudaSuccess) return cuda_fail(ea, "pca: Jacobi smem");
  int per_sm = 0;
  ea = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, bj_apply_kernel, 256, ap_smem);
  if (ea != cudaSuccess) return cuda_fail(ea, "pca: Jacobi occupancy");
  if (per_sm < 1) per_sm = 1;
  const int64_t ntiles = (int64_t)np * np - np + (int64_t)(n / kJS) * np;
  int64_t ap_blocks = (int64_t)num_sms() * per_sm;
  if (ap_blocks > ntiles) ap_blocks = ntiles;
  int sweep = 0;
  bool converged = false;
  const double tol2 = 0x1p-40;  // (2^-20)^2
  double prev_off = -1.0;
  for (sweep = 1; sweep <= kJacobiMaxSweeps && !converged; ++sweep) {
    for (int t = 0; t < nb - 1; ++t) {
      bj_sub_kernel<<<np, kSubThreads, 0, s>>>(A0, n, t, Qbuf);
      if (ap_blocks > 0) bj_apply_kernel<<<(unsigned)ap_blocks, 256, ap_smem, s>>>(A0, V0, n, t, Qbuf);
    }
    count_launch(2 * (nb - 1));
    cudaError_t e = cudaMemsetAsync(acc, 0, 2 * sizeof(double), s);
    if (e != cudaSuccess) return cuda_fail(e, "pca: clear norms");
    int nbk = (int)(((int64_t)n * n + 255) / 256);
    if (nbk > 4 * num_sms()) nbk = 4 * num_sms();
    jacobi_offnorm_kernel<<<nbk, 256, 0, s>>>(A0, n, acc);
    count_launch();
    double h[2];
    e = cudaMemcpyAsync(h, acc, sizeof(h), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e, "pca: Jacobi sweep");
    // converged: off(A) <= 2^-20 ||A||_F, or off(A) already below 2^-16 ||A||_F
    // and no longer halving from one sweep to the next (the fp32 floor)
    converged = h[0] <= tol2 * (h[0] + h[1]) ||
                (prev_off >= 0.0 && h[0] >= 0.25 * prev_off && h[0] <= 0x1p-32 * (h[0] + h[1]));
    prev_off = h[0];
  }
  if (sweeps_out) *sweeps_out = sweep - 1;
  if (!converged) return fail(HME_EINTERNAL, "pca: Jacobi did not converge in %d sweeps", kJacobiMaxSweeps);
  const size_t rank_smem = (size_t)g.d * sizeof(float);
  if (rank_smem > 48 * 1024) {
    cudaError_t ea = cudaFuncSetAttribute(pca_rank_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)rank_smem);
    if (ea != cudaSuccess) return cuda_fail(ea, "pca: rank smem");
  }
  pca_rank_kernel<<<1, 1024, rank_smem, s>>>(A0, n, g.d, g.r, order, variances);
  pca_components_kernel<<<g.r, 256, 0, s>>>(V0, n, g.d, order, W);
  count_launch(2);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "pca: components");
  return HME_OK;
}

cudaError_t launch_pca_zoff(const float *mean, const float *W, int d, int r, int Kp, float *zoff, cudaStream_t s) {
  pca_zoff_kernel<<<Kp, 256, 0, s>>>(mean, W, d, r, zoff);
  count_launch();
  return cudaGetLastError();
}

}  // namespace hme
