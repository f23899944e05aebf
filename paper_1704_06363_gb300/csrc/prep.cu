// prep.cu -- operand preparation for the tensor-core assign step.
//
// The assign step evaluates ||x - c||^2 = ||x||^2 - 2 x.c + ||c||^2 (the
// expansion of the distance in Eq. 2).  This file makes the pieces that are
// not the dot product:
//   prep_features  once per feature set: for fp32 features the bf16 split
//                  x_eff = hi + lo with hi = bf16_rn(x), lo = bf16_rn(x - hi),
//                  stored row-major with a 16-byte-aligned row stride for TMA,
//                  and xn[i] = ||x_eff,i||^2 of exactly those values; for bf16
//                  features xn[i] = ||x_i||^2.  One warp per row, 16-byte
//                  vector loads, read once (HBM-bound).
//                  fp32 features read as tf32 operands (several N-chunks)
//                  need only xn[i] = ||x_i||^2 of the fp32 values.
//   prep_centres   every iteration: bf16(c) (bf16 features) or the split
//                  ch, cl (fp32 features), and cn[k] = ||c_eff||^2 of exactly
//                  the values the MMA consumes; for tf32 operands c rounded to
//                  tf32 (cvt.rna) and cn[k] = ||c||^2 of the fp32 centre (the
//                  distance is taken to the fp32 centre; the operand rounding
//                  enters the near-tie bound); cn = +inf for padding centres;
//                  max_k cn[k] goes to the workspace header (error bound of the
//                  assign step's near-tie test).
#include "hme_common.cuh"

namespace hme {

namespace {

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ float4 ld_stream_f4(const float *p) {
  float4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.f32 {%0,%1,%2,%3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ void split_bf16(float x, __nv_bfloat16 &hi, __nv_bfloat16 &lo) {
  hi = __float2bfloat16_rn(x);
  lo = __float2bfloat16_rn(x - __bfloat162float(hi));
}

// fp32 features, 16-byte vectors (d % 4 == 0, ldx % 4 == 0, 16-byte aligned base).
__global__ void __launch_bounds__(256) prep_f32_vec_kernel(const float *__restrict__ X, int64_t N, int d,
                                                           int64_t ldx, int ldp, float *__restrict__ xn,
                                                           __nv_bfloat16 *__restrict__ xhi,
                                                           __nv_bfloat16 *__restrict__ xlo) {
  const int lane = threadIdx.x & 31;
  const int64_t w0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int d4 = d >> 2;
  for (int64_t row = w0; row < N; row += nw) {
    const float *xr = X + row * ldx;
    __nv_bfloat16 *hr = xhi + row * (int64_t)ldp;
    __nv_bfloat16 *lr = xlo + row * (int64_t)ldp;
    float s = 0.0f;
    for (int j = lane; j < d4; j += 32) {
      const float4 v = ld_stream_f4(xr + 4 * j);
      __nv_bfloat16 h[4], l[4];
      split_bf16(v.x, h[0], l[0]);
      split_bf16(v.y, h[1], l[1]);
      split_bf16(v.z, h[2], l[2]);
      split_bf16(v.w, h[3], l[3]);
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        const float e = __bfloat162float(h[t]) + __bfloat162float(l[t]);  // exact in fp32
        s = fmaf(e, e, s);
      }
      *reinterpret_cast<uint2 *>(hr + 4 * j) = *reinterpret_cast<const uint2 *>(h);
      *reinterpret_cast<uint2 *>(lr + 4 * j) = *reinterpret_cast<const uint2 *>(l);
    }
    s = warp_sum(s);
    if (lane == 0) xn[row] = s;
  }
}

// fp32 features, any layout.
__global__ void __launch_bounds__(256) prep_f32_scalar_kernel(const float *__restrict__ X, int64_t N, int d,
                                                              int64_t ldx, int ldp, float *__restrict__ xn,
                                                              __nv_bfloat16 *__restrict__ xhi,
                                                              __nv_bfloat16 *__restrict__ xlo) {
  const int lane = threadIdx.x & 31;
  const int64_t w0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t row = w0; row < N; row += nw) {
    float s = 0.0f;
    for (int j = lane; j < d; j += 32) {
      const float v = X[row * ldx + j];
      __nv_bfloat16 h, l;
      split_bf16(v, h, l);
      const float e = __bfloat162float(h) + __bfloat162float(l);
      s = fmaf(e, e, s);
      xhi[row * (int64_t)ldp + j] = h;
      xlo[row * (int64_t)ldp + j] = l;
    }
    s = warp_sum(s);
    if (lane == 0) xn[row] = s;
  }
}

// fp32 features read as tf32 operands: only the norms of the fp32 rows.
template <bool VEC>
__global__ void __launch_bounds__(256) prep_f32_norm_kernel(const float *__restrict__ X, int64_t N, int d,
                                                            int64_t ldx, float *__restrict__ xn) {
  const int lane = threadIdx.x & 31;
  const int64_t w0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t row = w0; row < N; row += nw) {
    const float *xr = X + row * ldx;
    float s = 0.0f;
    if (VEC) {  // d % 4 == 0, ldx % 4 == 0 and a 16-byte aligned base
      for (int j = lane; j < d / 4; j += 32) {
        const float4 v = ld_stream_f4(xr + 4 * j);
        s = fmaf(v.x, v.x, s);
        s = fmaf(v.y, v.y, s);
        s = fmaf(v.z, v.z, s);
        s = fmaf(v.w, v.w, s);
      }
    } else {
      for (int j = lane; j < d; j += 32) {
        const float v = __ldg(xr + j);
        s = fmaf(v, v, s);
      }
    }
    s = warp_sum(s);
    if (lane == 0) xn[row] = s;
  }
}

__device__ __forceinline__ float round_tf32(float x) {
  uint32_t r;
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
  return __uint_as_float(r);
}

// bf16 features: only the norms (the MMA reads X itself).
__global__ void __launch_bounds__(256) prep_bf16_kernel(const __nv_bfloat16 *__restrict__ X, int64_t N, int d,
                                                        int64_t ldx, float *__restrict__ xn) {
  const int lane = threadIdx.x & 31;
  const int64_t w0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int d8 = d >> 3;  // ldx % 8 == 0 and a 16-byte aligned base are checked on the host
  if (d8 <= 32 && 8 * d8 == d) {
    // at most one 16-byte vector per lane and row: four rows in flight per
    // warp (the same per-row arithmetic as the general loop below)
    for (int64_t r0 = w0; r0 < N; r0 += 4 * nw) {
      uint4 u[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int64_t row = r0 + k * nw;
        u[k] = make_uint4(0u, 0u, 0u, 0u);
        if (row < N && lane < d8)
          asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                       : "=r"(u[k].x), "=r"(u[k].y), "=r"(u[k].z), "=r"(u[k].w)
                       : "l"(X + row * ldx + 8 * lane));
      }
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int64_t row = r0 + k * nw;
        const __nv_bfloat162 *h2 = reinterpret_cast<const __nv_bfloat162 *>(&u[k]);
        float s = 0.0f;
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const float2 f = __bfloat1622float2(h2[t]);
          s = fmaf(f.x, f.x, s);
          s = fmaf(f.y, f.y, s);
        }
        s = warp_sum(s);
        if (lane == 0 && row < N) xn[row] = s;
      }
    }
    return;
  }
  for (int64_t row = w0; row < N; row += nw) {
    const __nv_bfloat16 *xr = X + row * ldx;
    float s = 0.0f;
    for (int j = lane; j < d8; j += 32) {
      uint4 u;
      asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                   : "=r"(u.x), "=r"(u.y), "=r"(u.z), "=r"(u.w)
                   : "l"(xr + 8 * j));
      const __nv_bfloat162 *h2 = reinterpret_cast<const __nv_bfloat162 *>(&u);
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        const float2 f = __bfloat1622float2(h2[t]);
        s = fmaf(f.x, f.x, s);
        s = fmaf(f.y, f.y, s);
      }
    }
    for (int j = 8 * d8 + lane; j < d; j += 32) {
      const float f = __bfloat162float(xr[j]);
      s = fmaf(f, f, s);
    }
    s = warp_sum(s);
    if (lane == 0) xn[row] = s;
  }
}

// Centres: one block per centre row k < Kp, the row's elements strided over
// the block's threads (several loads in flight per thread), then a block sum
// of the squared effective values.
constexpr int kPrepCThreads = 256;

__global__ void __launch_bounds__(kPrepCThreads) prep_centres_kernel(const float *__restrict__ C, int K, int Kp,
                                                                     int d, int ldp, int nprod, bool tf32,
                                                                     void *__restrict__ chi_raw,
                                                                     __nv_bfloat16 *__restrict__ clo,
                                                                     float *__restrict__ cn, Header *hdr) {
  // one warp per centre; the block's largest norm goes to cn_max once
  __nv_bfloat16 *chi = static_cast<__nv_bfloat16 *>(chi_raw);
  float *ct = static_cast<float *>(chi_raw);
  __shared__ float wmax[kPrepCThreads / 32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  float bmax = 0.0f;
  for (int k = blockIdx.x * (kPrepCThreads / 32) + warp; k < Kp; k += gridDim.x * (kPrepCThreads / 32)) {
    if (k >= K) {
      if (lane == 0) cn[k] = INFINITY;
      continue;
    }
    float s = 0.0f;
#pragma unroll 4
    for (int j = lane; j < d; j += 32) {
      const float c = __ldg(C + (int64_t)k * d + j);
      float ce;
      if (tf32) {
        ct[(int64_t)k * ldp + j] = round_tf32(c);
        ce = c;
      } else if (nprod == 1) {
        const __nv_bfloat16 bv = __float2bfloat16_rn(c);
        chi[(int64_t)k * ldp + j] = bv;
        ce = __bfloat162float(bv);
      } else {
        __nv_bfloat16 h, l;
        split_bf16(c, h, l);
        chi[(int64_t)k * ldp + j] = h;
        clo[(int64_t)k * ldp + j] = l;
        ce = __bfloat162float(h) + __bfloat162float(l);  // exact in fp32
      }
      s = fmaf(ce, ce, s);
    }
    s = warp_sum(s);
    if (lane == 0) cn[k] = s;
    bmax = fmaxf(bmax, s);
  }
  if (lane == 0) wmax[warp] = bmax;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.0f;
    for (int w = 0; w < kPrepCThreads / 32; ++w) t = fmaxf(t, wmax[w]);
    atomicMax(&hdr->cn_max_bits, __float_as_uint(t));  // t >= 0: integer order is float order
  }
}

}  // namespace

cudaError_t launch_prep_features(const void *X, int64_t N, int d, int64_t ldx, int dtype, const AssignGeom &g,
                                 float *xn, __nv_bfloat16 *xhi, __nv_bfloat16 *xlo, cudaStream_t s) {
  if (N == 0) return cudaSuccess;
  const int64_t want = (N + 7) / 8;  // 8 warps per block, one row per warp per pass
  int64_t blocks = (int64_t)num_sms() * 8;
  if (blocks > want) blocks = want;
  if (dtype == HME_F32) {
    const bool vec = (d % 4 == 0) && (ldx % 4 == 0) && ((reinterpret_cast<uintptr_t>(X) & 15u) == 0);
    const float *Xf = static_cast<const float *>(X);
    if (g.tf32 && vec)
      prep_f32_norm_kernel<true><<<(unsigned)blocks, 256, 0, s>>>(Xf, N, d, ldx, xn);
    else if (g.tf32)
      prep_f32_norm_kernel<false><<<(unsigned)blocks, 256, 0, s>>>(Xf, N, d, ldx, xn);
    else if (vec)
      prep_f32_vec_kernel<<<(unsigned)blocks, 256, 0, s>>>(Xf, N, d, ldx, g.ldp, xn, xhi, xlo);
    else
      prep_f32_scalar_kernel<<<(unsigned)blocks, 256, 0, s>>>(Xf, N, d, ldx, g.ldp, xn, xhi, xlo);
  } else {
    prep_bf16_kernel<<<(unsigned)blocks, 256, 0, s>>>(static_cast<const __nv_bfloat16 *>(X), N, d, ldx, xn);
  }
  count_launch();
  return cudaGetLastError();
}

cudaError_t launch_prep_centres(const float *C, const AssignGeom &g, void *chi, __nv_bfloat16 *clo, float *cn,
                                Header *hdr, cudaStream_t s) {
  const int per = kPrepCThreads / 32;  // centres per block and pass
  const int blocks = std::min((g.Kp + per - 1) / per, num_sms() * 4);
  prep_centres_kernel<<<blocks, kPrepCThreads, 0, s>>>(C, g.K, g.Kp, g.d, g.ldc, g.nprod, g.tf32, chi, clo, cn, hdr);
  count_launch();
  return cudaGetLastError();
}

}  // namespace hme
