// assign.cu -- fused nearest-centre assignment (Eq. 2, Section 2) on the
// sm_103a tensor cores.
//
// For a tile of 128 rows and a chunk of BN centres the kernel forms the dot
// products x.c with tcgen05.mma (bf16 operands, fp32 accumulator in TMEM),
// then four epilogue warps read the accumulator rows back with tcgen05.ld and
// keep, per row, the smallest and second-smallest  ||c||^2 - 2 x.c  and the
// index of the smallest (ties to the lower index because columns are scanned
// in ascending order and the comparison is strict).  Nothing of size N x K is
// ever written: per row the kernel emits a label, the distance to the chosen
// centre and, for near ties, a re-score request.
//
// Operands: for bf16 features, A = X (bf16) and B = bf16(C).  fp32 features
// with several N-chunks (K > 256, where the assign step is tensor-bound) are
// read by TMA as they are and multiplied as tf32 (kind::tf32: 10-bit
// significands, one product per k-step, 32 elements per 128-byte k-block)
// against tf32-rounded centres; the operand rounding, |x - x_tf32| <= 2^-10
// |x| and |c - c_tf32| <= 2^-11 |c| elementwise, enters the near-tie bound as
// a term 6.002 * 2^-10 ||x|| max ||c|| (twice the error of each of the two
// distances, 2 |x.c - x'.c'| <= 3.001 * 2^-10 ||x|| ||c||).  Otherwise fp32
// features use the split x = xh + xl, c = ch + cl (all bf16, 16 significant bits
// together) gives x_eff.c_eff = xh.ch + xh.cl + xl.ch + xl.cl.  The kernel
// issues the first three (three MMAs per k-step): |xl| <= 2^-8 (1 + 2^-8) |x|
// elementwise and likewise for cl, so the dropped xl.cl is at most
// 2^-16 (1 + 2^-8)^2 ||x|| ||c|| and enters the near-tie bound as its own
// term.  With ||x_eff||^2 and ||c_eff||^2 from the same split values the
// computed distance is ||x_eff - c_eff||^2 + 2 xl.cl up to fp32 accumulation;
// ||x_eff - c_eff||^2 differs from ||x - c||^2 by O(2^-16 |x - c| (|x| + |c|))
// per element.
//
// Warp roles (one CTA per SM, persistent over row tiles):
//   warp 0      TMA producer: A and B k-blocks into an S-stage ring,
//   warp 1      TMEM allocator and single-thread MMA issuer,
//   warps 2..   epilogue; warp w reads TMEM lanes 32*(w%4) .. 32*(w%4)+31,
//               CS warps per lane quarter and row tile, each scanning its
//               share of every chunk's columns.
// The accumulator is double-buffered in TMEM so the epilogue of one chunk
// overlaps the MMAs of the next.  Every wait is bounded (see
// mbar_wait_bounded); on expiry the kernel records HME_ETIMEOUT and ends.
#include "hme_common.cuh"

#include <cmath>
#include <cstdio>
#include <mutex>

namespace hme {

namespace {

struct AssignParams {
  int64_t N;
  int num_kb;          // k-blocks of 64 elements along d
  int BN, nchunks;
  int num_tiles;
  int stages;
  uint32_t a_bytes;    // one A operand per stage (128 rows x 128 bytes)
  uint32_t b_bytes;    // one B operand per stage (BN rows x 128 bytes)
  uint32_t stage_bytes;
  uint32_t tmem_cols;  // allocated TMEM columns
  uint32_t acc_stride; // columns between accumulator buffers
  int nbuf;            // accumulator buffers (2: epilogue overlaps the next MMAs)
  uint32_t a_res_bytes;  // resident A region (0 unless the A rows stay resident)
  // in-kernel split of fp32 features (assign_split_kernel)
  int sb_stages;          // centre (B) stages
  int st_stages;          // split A stages in tensor memory
  uint32_t b_stage_bytes; // one B stage (hi and lo operands)
  uint32_t a_col0;        // first TMEM column of the A stages
  int wide;               // 2 BN <= 256: xh.[ch; cl] as one N = 2 BN MMA (accumulator columns j and BN + j add up)
  int write_split;  // also store the split rows (tensor maps tmOh, tmOl) and their norms (xn_out)
  float *xn_out;
  float *z_out;     // projection mode: z_ij = x_i.c_j - cn_j for j < zcols, rows of pitch ldz (no argmin)
  int64_t ldz;
  int zcols;
  int zvec;         // z_out 16-byte aligned and ldz % 4 == 0: float4 stores
  const float *xn;
  const float *cn;     // Kp entries, +inf past K
  int32_t *labels;
  float *mind;
  Header *hdr;
  int32_t *flagged;    // (row, best, runner-up) of near-tie rows with two candidates
  int32_t *full_rows;  // near-tie rows to compare with all K centres
  uint64_t limit_ns;
  float err_acc;    // ceil(d/16) * nprod * 2^-22 + 2^-20: accumulation + epilogue rounding
  float err_split;  // 2^-14 for split fp32 operands, else 0
  float err_ll;     // 1.0625 * 2^-14 for split fp32 operands (the dropped xl.cl), else 0
  // small batches (lean scan only): the N-chunks of a row tile are spread over
  // `slices` CTAs of cps chunks each; each writes its row states to part and
  // assign_merge_kernel finishes the rows
  int slices, cps;
  float4 *part;     // [N][slices]: best, runner-up, third bound, centres of best and runner-up (bits)
};

constexpr uint32_t kWhereProducer = 1, kWhereMma = 2, kWhereMmaAcc = 3, kWhereEpi = 4, kWhereXchg = 6;

// One group of 16 accumulator columns of one row: v_j = ||c_j||^2 - 2 x.c_j.
// The running best three values (and the indices of the best two) change only
// when the group's minimum is below the third best, which after the first few
// groups is rare; that test is one compare per 16 columns.
__device__ __forceinline__ void epilogue_group(const uint32_t (&r)[16], const float *cn16, int k0, float &best1,
                                               float &best2, float &best3, int &idx1, int &idx2) {
  float v[16];
  const float4 *c4 = reinterpret_cast<const float4 *>(cn16);
  float m = INFINITY;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const float4 cc = c4[q];
    v[4 * q + 0] = fmaf(-2.0f, __uint_as_float(r[4 * q + 0]), cc.x);
    v[4 * q + 1] = fmaf(-2.0f, __uint_as_float(r[4 * q + 1]), cc.y);
    v[4 * q + 2] = fmaf(-2.0f, __uint_as_float(r[4 * q + 2]), cc.z);
    v[4 * q + 3] = fmaf(-2.0f, __uint_as_float(r[4 * q + 3]), cc.w);
    m = fminf(m, fminf(fminf(v[4 * q], v[4 * q + 1]), fminf(v[4 * q + 2], v[4 * q + 3])));
  }
  if (m < best3) {
#pragma unroll
    for (int j = 0; j < 16; ++j) {
      const float x = v[j];
      if (x < best1) {
        best3 = best2;
        best2 = best1;
        idx2 = idx1;
        best1 = x;
        idx1 = k0 + j;
      } else if (x < best2) {
        best3 = best2;
        best2 = x;
        idx2 = k0 + j;
      } else if (x < best3) {
        best3 = x;
      }
    }
  }
}

// Lean variant for many centres (several N-chunks): per column
// v = ||c||^2 - 2 x.c, then runner-up = min(runner-up, max(best, v)) and
// best = min(best, v) -- three ALU instructions.  The best's column is found
// only in a group that improved the best (after the first groups, rarely: a
// warp-uniform branch), as the first column of the group equal to the new
// best, so ties keep the lowest index.
__device__ __forceinline__ void lean_group(const uint32_t (&r)[16], const float *cn16, int k0, float &b1, float &b2,
                                           int &i1) {
  const float4 *c4 = reinterpret_cast<const float4 *>(cn16);
  const float before = b1;
  float v[16];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const float4 cc = c4[q];
    const float cq[4] = {cc.x, cc.y, cc.z, cc.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int j = 4 * q + e;
      v[j] = fmaf(-2.0f, __uint_as_float(r[j]), cq[e]);
      b2 = fminf(b2, fmaxf(b1, v[j]));
      b1 = fminf(b1, v[j]);
    }
  }
  if (b1 < before) {  // the first column of the group that holds the new best
    int jl = 15;
#pragma unroll
    for (int j = 14; j >= 0; --j) jl = (v[j] == b1) ? j : jl;
    i1 = k0 + jl;
  }
}

// Branch-free top three for many centres with tf32 operands (whose wider
// near-tie bound makes near ties common): per column v = ||c||^2 - 2 x.c,
// the three smallest values and the indices of the best two, so that a near
// tie with exactly two candidates is re-scored on those two only.  Ties keep
// the lower index (columns ascend, comparisons are strict).
__device__ __forceinline__ void top3_group(const uint32_t (&r)[16], const float *cn16, int k0, float &b1, float &b2,
                                           float &b3, int &i1, int &i2) {
  const float4 *c4 = reinterpret_cast<const float4 *>(cn16);
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const float4 cc = c4[q];
    const float cq[4] = {cc.x, cc.y, cc.z, cc.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int j = k0 + 4 * q + e;
      const float v = fmaf(-2.0f, __uint_as_float(r[4 * q + e]), cq[e]);
      const bool lt1 = v < b1, lt2 = v < b2;
      b3 = fminf(b3, fmaxf(b2, v));
      b2 = fminf(b2, fmaxf(b1, v));
      i2 = lt1 ? i1 : (lt2 ? j : i2);
      i1 = lt1 ? j : i1;
      b1 = fminf(b1, v);
    }
  }
}

// Insert (v, i) into a top-three state (value, then index order).
__device__ __forceinline__ void insert_top3(float v, int i, float &b1, float &b2, float &b3, int &i1, int &i2) {
  if (v < b1 || (v == b1 && i < i1)) {
    b3 = b2;
    b2 = b1;
    i2 = i1;
    b1 = v;
    i1 = i;
  } else if (v < b2 || (v == b2 && i < i2)) {
    b3 = b2;
    b2 = v;
    i2 = i;
  } else {
    b3 = fminf(b3, v);
  }
}

// The result of one row's scan: label, distance, and for a near tie a
// re-score request.  A centre whose tensor-core distance is within E of the
// best could be the true nearest one.  E bounds the error of a difference of
// two computed distances: each fp32 accumulation step of x.c errs by at most
// one ulp of the accumulator (|x.c| <= (||x||^2 + ||c||^2) / 2), the split
// operands of fp32 features by 2^-16 per element, and the epilogue adds a few
// roundings; the dropped xl.cl moves each distance by at most
// 2^-15 (1 + 2^-8)^2 ||x|| ||c||.  Such rows are queued for an exact
// comparison: of the two candidates, or of all K when a third centre is also
// within E (or, in the lean scan, whenever the runner-up is).  Returns the
// row's share of the objective estimate (0 for queued rows: the re-score adds
// theirs).
// Merge of two lean row states, each (b1, i1): best value and its centre,
// b2: the exact runner-up value, i2: its centre or -1 when unknown, b3: a
// lower bound of the third smallest value.  The best is the lexicographic
// minimum over (value, centre); the runner-up is the loser's best, whose
// centre is known, when that is below the winner's runner-up -- and the third
// is then min(winner's b2, loser's b2) exactly -- else the winner's runner-up
// (its centre as the winner knew it) with third >= min(winner's b3, loser's b1).
// A fresh lean scan state is (b1, i1, b2, -1, b2).
__device__ __forceinline__ void lean_merge(float &b1, int &i1, float &b2, int &i2, float &b3, float c1, int j1,
                                           float c2, int j2, float c3) {
  const bool other = c1 < b1 || (c1 == b1 && j1 < i1);
  const float w2 = other ? c2 : b2, w3 = other ? c3 : b3, l1 = other ? b1 : c1, l2 = other ? b2 : c2;
  const int wk = other ? j2 : i2, li = other ? i1 : j1;
  if (other) {
    b1 = c1;
    i1 = j1;
  }
  if (l1 < w2) {
    b2 = l1;
    i2 = li;
    b3 = fminf(w2, l2);
  } else {
    b2 = w2;
    i2 = wk;
    b3 = fminf(w3, l1);
  }
}

template <bool LEAN>
__device__ __forceinline__ double finish_row(const AssignParams &p, int64_t row, float xr, float best1, float best2,
                                             float best3, int idx1, int idx2, float cn_max, float sqrt_cn_max) {
  const float D1 = xr + best1;
  const float D2 = xr + best2;
  const float D3 = xr + best3;
  const float md = fmaxf(D1, 0.0f);
  p.labels[row] = idx1;
  if (p.mind) p.mind[row] = md;
  const float sqrt_xr = sqrtf(xr);
  const float E = p.err_acc * (xr + cn_max) + p.err_split * (sqrt_xr + sqrt_cn_max) * sqrtf(fmaxf(D2, 0.0f)) +
                  p.err_ll * sqrt_xr * sqrt_cn_max;
  const bool near2 = (best2 < INFINITY) && ((D2 - D1) <= E);
  if (!near2) return (double)md;
  // lean scan: two candidates only when the runner-up's centre is known and
  // the third value's lower bound is beyond E
  const bool near3 = (LEAN && idx2 < 0) || ((best3 < INFINITY) && ((D3 - D1) <= E));
  if (near3) {
    const uint32_t slot = atomicAdd(&p.hdr->rescore_full_count, 1u);
    p.full_rows[slot] = (int32_t)row;
  } else {
    const uint32_t slot = atomicAdd(&p.hdr->rescore_count, 1u);
    p.flagged[3 * slot + 0] = (int32_t)row;
    p.flagged[3 * slot + 1] = idx1;
    p.flagged[3 * slot + 2] = idx2;
  }
  return 0.0;
}

// The fused assign kernel.
//   NPROD  1: bf16 operands; 3: fp32 features as bf16 hi/lo pairs (three products)
//   LEAN   several N-chunks: lean epilogue scan (best, index, runner-up)
//   MT     row tiles of 128 per CTA sharing each B (centre) stage: 1 or 2
//   ARES   the CTA's A rows (all k-blocks) stay resident in shared memory for
//          all N-chunks; only B streams through the ring
//   CS     epilogue warps per (row tile, TMEM lane quarter), splitting each
//          chunk's columns in CS shares (1, 2 or 4); at the end of every tile
//          shares 1 .. CS-1 hand their per-row states to share 0 (through
//          shared memory, behind two bounded mbarriers), which merges them and
//          writes the row's result
//   TF32   fp32 operands read as tf32 (kind::tf32; k-blocks of 32 elements)
//   T3     (not LEAN) the top-three scan over several N-chunks: a near tie
//          with exactly two candidates is re-scored on those two only
// Threads: warp 0 TMA, warp 1 MMA, 4*MT*CS epilogue warps.
template <int NPROD, bool LEAN, int MT, bool ARES, int CS, bool TF32 = false, bool T3 = TF32>
__global__ void __launch_bounds__(64 + 128 * MT * CS, 1)
    assign_kernel(const __grid_constant__ CUtensorMap tmA0, const __grid_constant__ CUtensorMap tmA1,
                  const __grid_constant__ CUtensorMap tmB0, const __grid_constant__ CUtensorMap tmB1,
                  const AssignParams p) {
  constexpr int NOPS = (NPROD == 3) ? 2 : 1;  // operands per side (hi[, lo])
  constexpr int BMT = kBM * MT;               // rows per CTA tile
  constexpr int KBLK = TF32 ? 32 : kBK;       // elements per 128-byte k-block
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte alignment for the 128-byte swizzle atoms.
  const uint32_t raw_addr = smem_u32(smem_raw);
  const uint32_t base = (raw_addr + 1023u) & ~1023u;
  uint8_t *smem = smem_raw + (base - raw_addr);

  const int S = p.stages;
  const uint32_t ares = base;                         // resident A region (ARES)
  const uint32_t ring = base + p.a_res_bytes;         // stage ring
  uint8_t *ctrl = smem + p.a_res_bytes + (size_t)S * p.stage_bytes;
  uint64_t *full = reinterpret_cast<uint64_t *>(ctrl);
  uint64_t *empty = full + S;
  uint64_t *tfull = empty + S;
  uint64_t *tempty = tfull + 2;
  uint64_t *drain = tempty + 2;
  uint64_t *a_full = drain + 1;
  uint64_t *a_empty = a_full + 1;
  uint64_t *xfull = a_empty + 1;          // [2 slots][4 MT groups]: shares 1 .. CS-1 have written their states
  uint64_t *xempty = xfull + 8 * MT;      // [2 slots][4 MT groups]: ... and share 0 has read them
  uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(xempty + 8 * MT);
  // ||c||^2 of the chunk: kMaxBN / CS floats per epilogue warp (its columns)
  float *cnbuf = reinterpret_cast<float *>(ctrl + 512);
  // per-row states handed over to share 0: [2 slots][4 MT groups][CS - 1 shares][32 lanes]
  float4 *xchg = reinterpret_cast<float4 *>(ctrl + 512 + (size_t)4 * MT * kMaxBN * sizeof(float));

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int nbuf = p.nbuf;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_u32(&tfull[a]), 1);
      mbar_init(smem_u32(&tempty[a]), 4 * MT * CS);
    }
    mbar_init(smem_u32(drain), 1);
    mbar_init(smem_u32(a_full), 1);
    mbar_init(smem_u32(a_empty), 1);
    if (CS > 1)
      for (int b = 0; b < 8 * MT; ++b) {
        mbar_init(smem_u32(&xfull[b]), 32 * (CS - 1));
        mbar_init(smem_u32(&xempty[b]), 32);
      }
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tensormap(&tmA0);
    prefetch_tensormap(&tmB0);
    if (NPROD == 3) {
      prefetch_tensormap(&tmA1);
      prefetch_tensormap(&tmB1);
    }
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_holder), p.tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;

  // shared-memory addresses of the operands of stage s / k-block kb
  auto a_addr = [&](int op, int mt, int kb, uint32_t st) -> uint32_t {
    if (ARES) return ares + (uint32_t)(((mt * p.num_kb + kb) * NOPS + op)) * p.a_bytes;
    return st + (uint32_t)(op * MT + mt) * p.a_bytes;
  };
  auto b_addr = [&](int op, uint32_t st) -> uint32_t {
    return st + (ARES ? 0u : (uint32_t)(NOPS * MT) * p.a_bytes) + (uint32_t)op * p.b_bytes;
  };

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      const uint64_t pol_a = l2_policy_evict_first();
      const uint64_t pol_b = l2_policy_evict_last();
      uint32_t it = 0, tile_it = 0;
      int ps = 0;        // stage of iteration it
      uint32_t pph = 0;  // and its phase
      bool ok = true, a_pending = false;
      for (int item = blockIdx.x; item < p.num_tiles * p.slices && ok; item += gridDim.x, ++tile_it) {
        const int tile = item / p.slices;
        const int ch0 = (item % p.slices) * p.cps, ch1 = min(p.nchunks, ch0 + p.cps);
        const int32_t row0 = tile * BMT;
        if (ARES) {
          // the previous tile's MMAs must be done with the resident A rows
          if (!mbar_wait_bounded(smem_u32(a_empty), (tile_it & 1u) ^ 1u, p.limit_ns, p.hdr, kWhereProducer)) {
            ok = false;
            break;
          }
          const uint32_t ab = smem_u32(a_full);
          mbar_arrive_expect_tx(ab, p.a_res_bytes);
          for (int mt = 0; mt < MT; ++mt)
            for (int kb = 0; kb < p.num_kb; ++kb) {
              tma_load_2d(a_addr(0, mt, kb, 0), &tmA0, ab, kb * KBLK, row0 + mt * kBM, pol_a);
              if (NPROD == 3) tma_load_2d(a_addr(1, mt, kb, 0), &tmA1, ab, kb * KBLK, row0 + mt * kBM, pol_a);
            }
          a_pending = true;
        }
        for (int ch = ch0; ch < ch1 && ok; ++ch) {
          for (int kb = 0; kb < p.num_kb; ++kb, ++it) {
            // stage and phase of iteration it, by counting (no division)
            const int s = ps;
            const uint32_t ph = pph;
            if (++ps == S) {
              ps = 0;
              pph ^= 1u;
            }
            if (!mbar_wait_bounded(smem_u32(&empty[s]), ph ^ 1u, p.limit_ns, p.hdr, kWhereProducer)) {
              ok = false;
              break;
            }
            const uint32_t fb = smem_u32(&full[s]);
            mbar_arrive_expect_tx(fb, p.stage_bytes);
            const uint32_t st = ring + (uint32_t)s * p.stage_bytes;
            const int32_t kx = kb * KBLK;
            if (!ARES) {
              for (int mt = 0; mt < MT; ++mt) {
                tma_load_2d(a_addr(0, mt, kb, st), &tmA0, fb, kx, row0 + mt * kBM, pol_a);
                if (NPROD == 3) tma_load_2d(a_addr(1, mt, kb, st), &tmA1, fb, kx, row0 + mt * kBM, pol_a);
              }
            }
            tma_load_2d(b_addr(0, st), &tmB0, fb, kx, ch * p.BN, pol_b);
            if (NPROD == 3) tma_load_2d(b_addr(1, st), &tmB1, fb, kx, ch * p.BN, pol_b);
          }
        }
      }
      // Drain: every copy issued must land before the CTA may end.
      if (!ok) {
        const uint32_t issued = it;
        for (uint32_t j = (issued > (uint32_t)S ? issued - S : 0); j < issued; ++j)
          mbar_wait_bounded(smem_u32(&full[j % S]), (j / S) & 1u, 200000000ull, p.hdr, kWhereProducer);
        if (ARES && a_pending && tile_it > 0)
          mbar_wait_bounded(smem_u32(a_full), (tile_it - 1) & 1u, 200000000ull, p.hdr, kWhereProducer);
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      const uint32_t idesc = TF32 ? idesc_tf32_f32(kBM, (uint32_t)p.BN) : idesc_bf16_f32(kBM, (uint32_t)p.BN);
      uint32_t tile_it = 0;
      // Stage, accumulator buffer and their phases advance by counting, and
      // the operand descriptors by adding to their start-address field (in
      // 16-byte units: +2 per 16-element k-step; every offset here is a
      // multiple of 1024 bytes and shared addresses stay below 2^18), so the
      // one issuing thread spends few instructions per MMA.
      int s = 0;
      uint32_t ph = 0, a = 0, aph = 0;
      const uint64_t ring_desc = smem_desc_sw128(ring);
      const uint64_t ares_desc = smem_desc_sw128(ares);
      const uint64_t boff0 = (uint64_t)(((ARES ? 0u : (uint32_t)(NOPS * MT) * p.a_bytes)) >> 4);
      const uint64_t boff1 = boff0 + (uint64_t)(p.b_bytes >> 4);
      const uint64_t abytes16 = (uint64_t)(p.a_bytes >> 4);
      bool ok = true;
      for (int item = blockIdx.x; item < p.num_tiles * p.slices && ok; item += gridDim.x, ++tile_it) {
        const int ch0 = (item % p.slices) * p.cps, ch1 = min(p.nchunks, ch0 + p.cps);
        if (ARES) {
          if (!mbar_wait_bounded(smem_u32(a_full), tile_it & 1u, p.limit_ns, p.hdr, kWhereMma)) {
            ok = false;
            break;
          }
          tc_fence_after();
        }
        for (int ch = ch0; ch < ch1 && ok; ++ch) {
          if (!mbar_wait_bounded(smem_u32(&tempty[a]), aph ^ 1u, p.limit_ns, p.hdr, kWhereMmaAcc)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t dt = tmem_base + a * p.acc_stride;
          for (int kb = 0; kb < p.num_kb; ++kb) {
            if (!mbar_wait_bounded(smem_u32(&full[s]), ph, p.limit_ns, p.hdr, kWhereMma)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint64_t st_desc = ring_desc + (uint64_t)(((uint32_t)s * p.stage_bytes) >> 4);
            const uint64_t bd0 = st_desc + boff0, bd1 = st_desc + boff1;
#pragma unroll
            for (int mt = 0; mt < MT; ++mt) {
              const uint32_t dtm = dt + (uint32_t)(mt * p.BN);
              const uint64_t ad0 = ARES ? ares_desc + (uint64_t)((mt * p.num_kb + kb) * NOPS) * abytes16
                                        : st_desc + (uint64_t)mt * abytes16;
              const uint64_t ad1 = ARES ? ad0 + abytes16 : st_desc + (uint64_t)(MT + mt) * abytes16;
#pragma unroll
              for (int k = 0; k < kBK / 16; ++k) {
                const uint64_t dk = (uint64_t)(2 * k);
                if (TF32)
                  tc_mma_tf32(dtm, ad0 + dk, bd0 + dk, idesc, (kb > 0 || k > 0) ? 1u : 0u);
                else
                  tc_mma_bf16(dtm, ad0 + dk, bd0 + dk, idesc, (kb > 0 || k > 0) ? 1u : 0u);
                if (NPROD == 3) {
                  tc_mma_bf16(dtm, ad0 + dk, bd1 + dk, idesc, 1u);  // xh . cl
                  tc_mma_bf16(dtm, ad1 + dk, bd0 + dk, idesc, 1u);  // xl . ch
                }
              }
            }
            tc_commit(smem_u32(&empty[s]));  // frees the stage once these MMAs finish
            if (++s == S) {
              s = 0;
              ph ^= 1u;
            }
          }
          if (ok) tc_commit(smem_u32(&tfull[a]));  // accumulators of buffer a are complete
          if (++a == (uint32_t)nbuf) {
            a = 0;
            aph ^= 1u;
          }
        }
        if (ARES && ok) tc_commit(smem_u32(a_empty));  // the resident A rows may be replaced
      }
      if (!ok) {
        // Let the MMAs already issued finish before TMEM is released.
        tc_commit(smem_u32(drain));
        mbar_wait_bounded(smem_u32(drain), 0, 200000000ull, p.hdr, kWhereMma);
      }
    }
  } else {
    // ---------------- epilogue: argmin over the accumulator rows ----------------
    const int e = warp - 2;          // 0 .. 4*MT*CS-1
    const int q = warp & 3;          // TMEM lane quarter this warp may access
    const int mt = (e >> 2) % MT;    // which row tile (accumulator) of the CTA tile
    const int half = (e >> 2) / MT;  // which share of the chunk's columns
    const int pr = mt * 4 + q;       // the group of CS warps sharing these rows
    // columns [c0, c1) of every chunk; shares are multiples of 16 columns
    // (trailing shares may be empty when BN is small)
    const int cw = CS == 1 ? p.BN : ((p.BN + CS - 1) / CS + 15) / 16 * 16;
    const int c0 = half * cw;
    const int c1 = min(p.BN, c0 + cw);
    float *cb = cnbuf + e * (kMaxBN / CS);  // this warp's copy of ||c||^2 of its columns
    const float cn_max = __uint_as_float(*((volatile uint32_t *)&p.hdr->cn_max_bits));
    const float sqrt_cn_max = sqrtf(cn_max);
    const int row_in_tile = mt * kBM + q * 32 + lane;
    uint32_t acc_it = 0, tile_it = 0;
    bool ok = true;
    double obj = 0.0;
    // ||c||^2 of the next chunk is fetched into registers while the current
    // chunk is scanned; with a single chunk the buffer is filled once.
    constexpr int kCnRegs = kMaxBN / CS / 32;
    float cn_next[kCnRegs];
    auto fetch_cn = [&](int ch) {
#pragma unroll
      for (int r = 0; r < kCnRegs; ++r) {
        const int t = c0 + lane + 32 * r;
        cn_next[r] = (t < c1) ? __ldg(p.cn + ch * p.BN + t) : 0.0f;
      }
    };
    fetch_cn(((int)blockIdx.x % p.slices) * p.cps);  // the first item's first chunk
    bool cb_filled = false;
    for (int item = blockIdx.x; item < p.num_tiles * p.slices && ok; item += gridDim.x, ++tile_it) {
      const int tile = item / p.slices, slice = item % p.slices;
      const int ch0 = slice * p.cps, ch1 = min(p.nchunks, ch0 + p.cps);
      // the first chunk of this CTA's next work item (its scan prefetches that chunk's norms)
      const int next_ch0 = ((item + (int)gridDim.x) % p.slices) * p.cps;
      float best1 = INFINITY, best2 = INFINITY, best3 = INFINITY;
      int idx1 = 0, idx2 = 0;
      float lb1 = INFINITY, lb2 = INFINITY;  // second independent state of the lean scan (odd groups)
      int li1 = 0;
      float lb3 = INFINITY;  // ... and of the tf32 top-three scan
      int li2 = 0;
      const int64_t row = (int64_t)tile * BMT + row_in_tile;
      const float xr = (half == 0 && row < p.N) ? __ldg(p.xn + row) : 0.0f;  // in flight during the scan
      for (int ch = ch0; ch < ch1; ++ch, ++acc_it) {
        if (p.nchunks > 1 || !cb_filled) {
          __syncwarp();
#pragma unroll
          for (int r = 0; r < kCnRegs; ++r)
            if (c0 + lane + 32 * r < c1) cb[lane + 32 * r] = cn_next[r];
          __syncwarp();
          cb_filled = true;
          if (p.nchunks > 1) fetch_cn(ch + 1 < ch1 ? ch + 1 : next_ch0);
        }
        const uint32_t a = acc_it % (uint32_t)nbuf;
        const uint32_t aph = (acc_it / (uint32_t)nbuf) & 1u;
        if (!mbar_wait_bounded(smem_u32(&tfull[a]), aph, p.limit_ns, p.hdr, kWhereEpi)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t taddr =
            tmem_base + a * p.acc_stride + (uint32_t)(mt * p.BN) + ((uint32_t)(q * 32) << 16);
        const int kbase = ch * p.BN;
        // 16 columns per step; the next step's tcgen05.ld is in flight while this
        // step's distances are formed.
        uint32_t ra[16], rb[16];
        if (c0 < c1) {
          tmem_ld16(taddr + (uint32_t)c0, ra);
          tmem_ld_wait(ra);
        }
        for (int c = c0; c < c1; c += 32) {
          const bool more1 = c + 16 < c1, more2 = c + 32 < c1;
          const float *cbc = cb + (c - c0);
          if (more1) tmem_ld16(taddr + (uint32_t)(c + 16), rb);
          if (LEAN)
            lean_group(ra, cbc, kbase + c, best1, best2, idx1);
          else if (T3)
            top3_group(ra, cbc, kbase + c, best1, best2, best3, idx1, idx2);
          else
            epilogue_group(ra, cbc, kbase + c, best1, best2, best3, idx1, idx2);
          if (more1) {
            tmem_ld_wait(rb);
            if (more2) tmem_ld16(taddr + (uint32_t)(c + 32), ra);
            if (LEAN)
              lean_group(rb, cbc + 16, kbase + c + 16, lb1, lb2, li1);
            else if (T3)
              top3_group(rb, cbc + 16, kbase + c + 16, lb1, lb2, lb3, li1, li2);
            else
              epilogue_group(rb, cbc + 16, kbase + c + 16, best1, best2, best3, idx1, idx2);
            if (more2) tmem_ld_wait(ra);
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&tempty[a]));
      }
      if (!ok) break;
      if (LEAN) {  // merge the two lean states (even and odd 16-column groups)
        idx2 = -1;
        best3 = best2;
        lean_merge(best1, idx1, best2, idx2, best3, lb1, li1, lb2, -1, lb2);
      } else if (T3) {  // merge the two top-three states
        insert_top3(lb1, li1, best1, best2, best3, idx1, idx2);
        insert_top3(lb2, li2, best1, best2, best3, idx1, idx2);
        best3 = fminf(best3, lb3);
      }
      if (CS > 1) {
        // Hand-over of the other shares' states.  Two slots alternate by
        // tile; a slot is rewritten only after share 0 has read it.
        const uint32_t slot = tile_it & 1u, use = tile_it >> 1;
        const int b = (int)slot * 4 * MT + pr;
        float4 *xs = xchg + (b * (CS - 1)) * 32 + lane;
        if (half > 0) {
          if (!mbar_wait_bounded(smem_u32(&xempty[b]), (use & 1u) ^ 1u, p.limit_ns, p.hdr, kWhereXchg)) {
            ok = false;
            break;
          }
          // indices < 2^16 (K <= 16384): both fit one word (an unknown lean
          // runner-up centre, -1, as 0xffff)
          xs[(half - 1) * 32] = make_float4(
              best1, best2, best3, __uint_as_float((uint32_t)idx1 | (((uint32_t)idx2 & 0xffffu) << 16)));
          mbar_arrive(smem_u32(&xfull[b]));
          continue;
        }
        if (!mbar_wait_bounded(smem_u32(&xfull[b]), use & 1u, p.limit_ns, p.hdr, kWhereXchg)) {
          ok = false;
          break;
        }
        float4 os[CS > 1 ? CS - 1 : 1];
#pragma unroll
        for (int h = 0; h < CS - 1; ++h) os[h] = xs[h * 32];
        mbar_arrive(smem_u32(&xempty[b]));
        // The merged best is the lexicographic minimum over (value, index)
        // and the runner-up the smallest remaining value: independent of the
        // merge order.  (Whether the lean runner-up's centre is known depends
        // on it; that only chooses between the pair and the all-K re-score.)
#pragma unroll
        for (int h = 0; h < CS - 1; ++h) {
          const float4 o = os[h];
          const uint32_t oi = __float_as_uint(o.w);
          const int o1 = (int)(oi & 0xffffu), o2 = (int)(oi >> 16);
          if (LEAN) {
            lean_merge(best1, idx1, best2, idx2, best3, o.x, o1, o.y, o2 == 0xffff ? -1 : o2, o.z);
          } else {
            // insert the other share's best two (value, then index) and its third value
            auto insert = [&](float v, int i) {
              if (v < best1 || (v == best1 && i < idx1)) {
                best3 = best2;
                best2 = best1;
                idx2 = idx1;
                best1 = v;
                idx1 = i;
              } else if (v < best2 || (v == best2 && i < idx2)) {
                best3 = best2;
                best2 = v;
                idx2 = i;
              } else {
                best3 = fminf(best3, v);
              }
            };
            insert(o.x, o1);
            insert(o.y, o2);
            best3 = fminf(best3, o.z);
          }
        }
      }
      if (p.slices > 1) {
        // a slice of the centres: its row state goes to assign_merge_kernel
        if (LEAN && row < p.N)
          p.part[row * p.slices + slice] =
              make_float4(best1, best2, best3, __uint_as_float((uint32_t)idx1 | (((uint32_t)idx2 & 0xffffu) << 16)));
      } else if (row < p.N) {
        obj += finish_row<LEAN>(p, row, xr, best1, best2, best3, idx1, idx2, cn_max, sqrt_cn_max);
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) obj += __shfl_xor_sync(0xffffffffu, obj, o);
    if (lane == 0 && obj != 0.0) atomicAdd(&p.hdr->objective, obj);
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, p.tmem_cols);
  }
}

// Small batches: the lean row states of the centre slices (best value and
// centre, runner-up value and centre if known, third-value bound) merged per
// row -- a group of kMaxSlices lanes per row, one slice each, merged by
// shuffles (lean_merge gives the same state whichever side it runs on) --
// then the row finished as in the assign kernel (label, distance, near-tie
// queues, objective).
constexpr int kMergeRows = 256 / kMaxSlices;  // rows per block
__global__ void __launch_bounds__(256) assign_merge_kernel(const AssignParams p) {
  static_assert(kMaxSlices <= 32 && (32 % kMaxSlices) == 0, "a row's slices fit one warp");
  const float cn_max = __uint_as_float(*((volatile uint32_t *)&p.hdr->cn_max_bits));
  const float sqrt_cn_max = sqrtf(cn_max);
  const int g = threadIdx.x % kMaxSlices;  // slice of this lane
  const int64_t row = (int64_t)blockIdx.x * kMergeRows + threadIdx.x / kMaxSlices;
  float best1 = INFINITY, best2 = INFINITY, best3 = INFINITY;
  int idx1 = 0x7fffffff, idx2 = -1;
  if (row < p.N && g < p.slices) {
    const float4 v = p.part[row * p.slices + g];
    const uint32_t ii = __float_as_uint(v.w);
    best1 = v.x;
    best2 = v.y;
    best3 = v.z;
    idx1 = (int)(ii & 0xffffu);
    idx2 = (ii >> 16) == 0xffffu ? -1 : (int)(ii >> 16);
  }
#pragma unroll
  for (int o = kMaxSlices / 2; o > 0; o >>= 1) {
    const float o1 = __shfl_xor_sync(0xffffffffu, best1, o);
    const float o2 = __shfl_xor_sync(0xffffffffu, best2, o);
    const float o3 = __shfl_xor_sync(0xffffffffu, best3, o);
    const int oi = __shfl_xor_sync(0xffffffffu, idx1, o);
    const int ok = __shfl_xor_sync(0xffffffffu, idx2, o);
    lean_merge(best1, idx1, best2, idx2, best3, o1, oi, o2, ok, o3);
  }
  double obj = 0.0;
  if (g == 0 && row < p.N)
    obj = finish_row<true>(p, row, __ldg(p.xn + row), best1, best2, best3, idx1, idx2, cn_max, sqrt_cn_max);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) obj += __shfl_xor_sync(0xffffffffu, obj, o);
  if ((threadIdx.x & 31) == 0 && obj != 0.0) atomicAdd(&p.hdr->objective, obj);
}

// ---------------------------------------------------------------------------
// fp32 features split on the fly (one N-chunk, K <= 256)
// ---------------------------------------------------------------------------
// The same contraction as assign_kernel<3, false, 1, false>, with the bf16
// hi/lo split of x made inside the kernel instead of by a preparation pass:
// the fp32 rows arrive by TMA (two 128-row x 32-column boxes per 64-column
// k-block, 128-byte swizzle), four converter warps split them (x = xh + xl,
// both rounded to nearest even), sum ||xh + xl||^2 per row, and store xh and
// xl into tensor memory, where the MMA reads them as its A operand (row m in
// lane m, bf16 pairs along k per 32-bit column).  B (ch, cl) streams from
// shared memory as before.  HBM traffic per row is the fp32 row itself, read
// once per call; no split copy of X exists.
// Warps: 0 X producer, 1 TMEM allocator + MMA issuer, 2 B producer,
// 3-10 converters (two per TMEM lane quarter, taking alternate k-blocks, so
// that one converts while the other waits on its stores), 11-14 epilogue
// (warp w touches TMEM lanes 32 (w % 4) ..).
constexpr int kSplitWarps = 15;
constexpr int kConvFirst = 3, kEpiFirst = 11;
constexpr int kSplitThreads = 32 * kSplitWarps;
constexpr uint32_t kXBox = kBM * 32 * 4;  // 128 rows x 32 fp32 = 16 KB
constexpr uint32_t kXStage = 2 * kXBox;   // one 64-column k-block
constexpr uint32_t kWhereConv = 5;

// x0, x1 -> packed bf16 pair (x0 in the low half), rounded to nearest even
__device__ __forceinline__ uint32_t pack_bf16x2(float x0, float x1) {
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(x1), "f"(x0));
  return r;
}

__global__ void __launch_bounds__(kSplitThreads, 1)
    assign_split_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmB0,
                        const __grid_constant__ CUtensorMap tmB1, const __grid_constant__ CUtensorMap tmOh,
                        const __grid_constant__ CUtensorMap tmOl, const AssignParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw_addr = smem_u32(smem_raw);
  const uint32_t base = (raw_addr + 1023u) & ~1023u;
  uint8_t *smem = smem_raw + (base - raw_addr);

  const int SX = p.stages, SB = p.sb_stages, ST = p.st_stages;
  const uint32_t xring = base;
  const uint32_t bring = base + (uint32_t)SX * kXStage;
  uint8_t *ctrl = smem + (size_t)SX * kXStage + (size_t)SB * p.b_stage_bytes;
  uint64_t *x_full = reinterpret_cast<uint64_t *>(ctrl);
  uint64_t *x_empty = x_full + SX;
  uint64_t *b_full = x_empty + SX;
  uint64_t *b_empty = b_full + SB;
  uint64_t *a_full = b_empty + SB;
  uint64_t *a_empty = a_full + ST;
  uint64_t *tfull = a_empty + ST;
  uint64_t *tempty = tfull + 2;
  uint64_t *xn_full = tempty + 2;
  uint64_t *xn_empty = xn_full + 2;
  uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(xn_empty + 2);
  float *xn_buf = reinterpret_cast<float *>(ctrl + 512);  // [2 buffers][2 converter halves][128 rows]
  float *cnbuf = xn_buf + 4 * kBM;                         // [4][kMaxBN]

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int nbuf = p.nbuf;

  if (threadIdx.x == 0) {
    for (int i = 0; i < SX; ++i) {
      mbar_init(smem_u32(&x_full[i]), 1);
      mbar_init(smem_u32(&x_empty[i]), 4);
    }
    for (int i = 0; i < SB; ++i) {
      mbar_init(smem_u32(&b_full[i]), 1);
      mbar_init(smem_u32(&b_empty[i]), 1);
    }
    for (int i = 0; i < ST; ++i) {
      mbar_init(smem_u32(&a_full[i]), 4);
      mbar_init(smem_u32(&a_empty[i]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&tfull[i]), 1);
      mbar_init(smem_u32(&tempty[i]), 4);
      mbar_init(smem_u32(&xn_full[i]), 8);
      mbar_init(smem_u32(&xn_empty[i]), 4);
    }
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) prefetch_tensormap(&tmX);
  if (warp == 2 && lane == 0) {
    prefetch_tensormap(&tmB0);
    prefetch_tensormap(&tmB1);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_holder), p.tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;

  if (warp == 0) {
    // ---------------- X producer: fp32 k-blocks ----------------
    if (lane == 0) {
      const uint64_t pol = l2_policy_evict_first();
      uint32_t i = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < p.num_tiles && ok; tile += gridDim.x) {
        const int32_t row0 = tile * kBM;
        for (int kb = 0; kb < p.num_kb; ++kb, ++i) {
          const int s = i % SX;
          if (!mbar_wait_bounded(smem_u32(&x_empty[s]), ((i / SX) & 1u) ^ 1u, p.limit_ns, p.hdr, kWhereProducer)) {
            ok = false;
            break;
          }
          const uint32_t fb = smem_u32(&x_full[s]);
          mbar_arrive_expect_tx(fb, kXStage);
          const uint32_t st = xring + (uint32_t)s * kXStage;
          tma_load_2d(st, &tmX, fb, kb * kBK, row0, pol);
          tma_load_2d(st + kXBox, &tmX, fb, kb * kBK + 32, row0, pol);
        }
      }
      if (!ok)  // every copy issued must land before the CTA may end
        for (uint32_t j = (i > (uint32_t)SX ? i - SX : 0); j < i; ++j)
          mbar_wait_bounded(smem_u32(&x_full[j % SX]), (j / SX) & 1u, 200000000ull, p.hdr, kWhereProducer);
    }
  } else if (warp == 2) {
    // ---------------- B producer: centre k-blocks (hi, lo) ----------------
    if (lane == 0) {
      const uint64_t pol = l2_policy_evict_last();
      uint32_t i = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < p.num_tiles && ok; tile += gridDim.x) {
        for (int kb = 0; kb < p.num_kb; ++kb, ++i) {
          const int s = i % SB;
          if (!mbar_wait_bounded(smem_u32(&b_empty[s]), ((i / SB) & 1u) ^ 1u, p.limit_ns, p.hdr, kWhereProducer)) {
            ok = false;
            break;
          }
          const uint32_t fb = smem_u32(&b_full[s]);
          mbar_arrive_expect_tx(fb, p.b_stage_bytes);
          const uint32_t st = bring + (uint32_t)s * p.b_stage_bytes;
          tma_load_2d(st, &tmB0, fb, kb * kBK, 0, pol);
          tma_load_2d(st + p.b_bytes, &tmB1, fb, kb * kBK, 0, pol);
        }
      }
      if (!ok)
        for (uint32_t j = (i > (uint32_t)SB ? i - SB : 0); j < i; ++j)
          mbar_wait_bounded(smem_u32(&b_full[j % SB]), (j / SB) & 1u, 200000000ull, p.hdr, kWhereProducer);
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(kBM, (uint32_t)p.BN);
      const uint32_t idesc2 = idesc_bf16_f32(kBM, 2u * (uint32_t)p.BN);
      uint32_t i = 0, acc_it = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < p.num_tiles && ok; tile += gridDim.x, ++acc_it) {
        const uint32_t a = acc_it % (uint32_t)nbuf;
        if (!mbar_wait_bounded(smem_u32(&tempty[a]), ((acc_it / (uint32_t)nbuf) & 1u) ^ 1u, p.limit_ns, p.hdr,
                               kWhereMmaAcc)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t dt = tmem_base + a * p.acc_stride;
        for (int kb = 0; kb < p.num_kb; ++kb, ++i) {
          const int t = i % ST, sb = i % SB;
          if (!mbar_wait_bounded(smem_u32(&a_full[t]), (i / ST) & 1u, p.limit_ns, p.hdr, kWhereMma) ||
              !mbar_wait_bounded(smem_u32(&b_full[sb]), (i / SB) & 1u, p.limit_ns, p.hdr, kWhereMma)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t at = tmem_base + p.a_col0 + (uint32_t)t * 64u;
          const uint32_t bst = bring + (uint32_t)sb * p.b_stage_bytes;
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k) {
            const uint64_t bd0 = smem_desc_sw128(bst + k * 32);
            const uint64_t bd1 = smem_desc_sw128(bst + p.b_bytes + k * 32);
            if (p.wide) {
              // ch and cl are adjacent in the stage: one MMA over both (columns
              // 0..BN-1 get xh.ch, BN..2BN-1 get xh.cl), then xl.ch into 0..BN-1
              tc_mma_bf16_ts(dt, at + 8u * k, bd0, idesc2, (kb > 0 || k > 0) ? 1u : 0u);  // xh . [ch; cl]
              tc_mma_bf16_ts(dt, at + 32u + 8u * k, bd0, idesc, 1u);                       // xl . ch
            } else {
              tc_mma_bf16_ts(dt, at + 8u * k, bd0, idesc, (kb > 0 || k > 0) ? 1u : 0u);  // xh . ch
              tc_mma_bf16_ts(dt, at + 8u * k, bd1, idesc, 1u);                           // xh . cl
              tc_mma_bf16_ts(dt, at + 32u + 8u * k, bd0, idesc, 1u);                     // xl . ch
            }
          }
          tc_commit(smem_u32(&a_empty[t]));
          tc_commit(smem_u32(&b_empty[sb]));
        }
        if (ok) tc_commit(smem_u32(&tfull[a]));
      }
    }
  } else if (warp < kEpiFirst) {
    // ---------------- converters: fp32 rows -> bf16 hi/lo in TMEM ----------------
    const int q = warp & 3;
    const uint32_t half = (uint32_t)((warp - kConvFirst) >> 2);  // k-blocks i with i % 2 == half
    const int r = q * 32 + lane;  // row within the tile = TMEM lane
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    uint32_t i = 0, tile_it = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < p.num_tiles && ok; tile += gridDim.x, ++tile_it) {
      float xs = 0.0f;  // ||xh + xl||^2 of this row over this warp's k-blocks
      for (int kb = 0; kb < p.num_kb; ++kb, ++i) {
        if ((i & 1u) != half) continue;
        const int s = i % SX, t = i % ST;
        if (!mbar_wait_bounded(smem_u32(&x_full[s]), (i / SX) & 1u, p.limit_ns, p.hdr, kWhereConv) ||
            !mbar_wait_bounded(smem_u32(&a_empty[t]), ((i / ST) & 1u) ^ 1u, p.limit_ns, p.hdr, kWhereConv)) {
          ok = false;
          break;
        }
        tc_fence_after();
        uint32_t hi[32], lo[32];
        const uint32_t rowaddr = xring + (uint32_t)s * kXStage + (uint32_t)r * 128u;
#pragma unroll
        for (int box = 0; box < 2; ++box) {
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            const float4 v = ld_shared_f4(rowaddr + (uint32_t)box * kXBox + ((uint32_t)(c ^ (r & 7)) << 4));
            const float xv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const float x0 = xv[2 * h], x1 = xv[2 * h + 1];
              const uint32_t hp = pack_bf16x2(x0, x1);
              const float h0 = __uint_as_float(hp << 16), h1 = __uint_as_float(hp & 0xFFFF0000u);
              const uint32_t lp = pack_bf16x2(x0 - h0, x1 - h1);
              const float l0 = __uint_as_float(lp << 16), l1 = __uint_as_float(lp & 0xFFFF0000u);
              const float e0 = h0 + l0, e1 = h1 + l1;  // exact in fp32
              xs = fmaf(e0, e0, xs);
              xs = fmaf(e1, e1, xs);
              hi[box * 16 + 2 * c + h] = hp;
              lo[box * 16 + 2 * c + h] = lp;
            }
          }
        }
        const uint32_t at = tmem_base + lane_off + p.a_col0 + (uint32_t)t * 64u;
        if (p.write_split) {
          // Leave the split behind for later prepared calls: this thread has
          // read all of its row, so it overwrites the row in place (hi in the
          // first box, lo in the second, each a 64-column bf16 row in the same
          // 128-byte swizzle) and lane 0 stores the warp's 32 rows with TMA;
          // the stage is released once the bulk copies have read it.
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            const uint32_t off = (uint32_t)r * 128u + ((uint32_t)(c ^ (r & 7)) << 4);
            st_shared_u4(xring + (uint32_t)s * kXStage + off, hi[4 * c], hi[4 * c + 1], hi[4 * c + 2], hi[4 * c + 3]);
            st_shared_u4(xring + (uint32_t)s * kXStage + kXBox + off, lo[4 * c], lo[4 * c + 1], lo[4 * c + 2],
                         lo[4 * c + 3]);
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0 && (int64_t)tile * kBM + q * 32 < p.N) {  // rows past N are clipped by TMA
            const uint32_t src = xring + (uint32_t)s * kXStage + (uint32_t)q * 32u * 128u;
            tma_store_2d(&tmOh, src, kb * kBK, tile * kBM + q * 32);
            tma_store_2d(&tmOl, src + kXBox, kb * kBK, tile * kBM + q * 32);
            bulk_commit();
          }
          tmem_st16(at, hi);
          tmem_st16(at + 16u, hi + 16);
          tmem_st16(at + 32u, lo);
          tmem_st16(at + 48u, lo + 16);
          if (lane == 0) {
            bulk_wait_read_all();
            mbar_arrive(smem_u32(&x_empty[s]));
          }
        } else {
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&x_empty[s]));  // the fp32 stage may be refilled
          tmem_st16(at, hi);
          tmem_st16(at + 16u, hi + 16);
          tmem_st16(at + 32u, lo);
          tmem_st16(at + 48u, lo + 16);
        }
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&a_full[t]));
      }
      if (!ok) break;
      const uint32_t b = tile_it & 1u;
      if (!mbar_wait_bounded(smem_u32(&xn_empty[b]), ((tile_it >> 1) & 1u) ^ 1u, p.limit_ns, p.hdr, kWhereConv)) {
        ok = false;
        break;
      }
      xn_buf[(b * 2 + half) * kBM + r] = xs;
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&xn_full[b]));
    }
    if (p.write_split && lane == 0) bulk_wait_all();
  } else {
    // ---------------- epilogue: argmin over the accumulator rows ----------------
    const int q = warp & 3;
    const int e = warp - kEpiFirst;
    float *cb = cnbuf + e * kMaxBN;
    for (int t = lane; t < p.BN; t += 32) cb[t] = __ldg(p.cn + t);
    __syncwarp();
    const float cn_max = __uint_as_float(*((volatile uint32_t *)&p.hdr->cn_max_bits));
    const float sqrt_cn_max = sqrtf(cn_max);
    const int r = q * 32 + lane;
    uint32_t acc_it = 0;
    bool ok = true;
    double obj = 0.0;
    for (int tile = blockIdx.x; tile < p.num_tiles && ok; tile += gridDim.x, ++acc_it) {
      const uint32_t a = acc_it % (uint32_t)nbuf;
      const uint32_t b = acc_it & 1u;
      if (!mbar_wait_bounded(smem_u32(&tfull[a]), (acc_it / (uint32_t)nbuf) & 1u, p.limit_ns, p.hdr, kWhereEpi) ||
          !mbar_wait_bounded(smem_u32(&xn_full[b]), (acc_it >> 1) & 1u, p.limit_ns, p.hdr, kWhereEpi)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const float xr = xn_buf[(b * 2) * kBM + r] + xn_buf[(b * 2 + 1) * kBM + r];
      if (p.xn_out && (int64_t)tile * kBM + r < p.N) p.xn_out[(int64_t)tile * kBM + r] = xr;
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&xn_empty[b]));
      float best1 = INFINITY, best2 = INFINITY, best3 = INFINITY;
      int idx1 = 0, idx2 = 0;
      const uint32_t taddr = tmem_base + a * p.acc_stride + ((uint32_t)(q * 32) << 16);
      uint32_t ra[16], rb[16];
      if (p.z_out) {
        // projection: write x.c_j - cn_j (cn holds the per-column offsets)
        const int64_t row = (int64_t)tile * kBM + r;
        float *zr = p.z_out + row * p.ldz;
        for (int c = 0; c < p.BN; c += 16) {
          tmem_ld16(taddr + (uint32_t)c, ra);
          if (p.wide) tmem_ld16(taddr + (uint32_t)(p.BN + c), rb);
          tmem_ld_wait(ra);
          if (p.wide) {
            tmem_ld_wait(rb);
#pragma unroll
            for (int j = 0; j < 16; ++j) ra[j] = __float_as_uint(__uint_as_float(ra[j]) + __uint_as_float(rb[j]));
          }
          float z[16];
#pragma unroll
          for (int j = 0; j < 16; ++j) z[j] = __uint_as_float(ra[j]) - cb[c + j];
          if (row < p.N) {
            if (p.zvec && c + 16 <= p.zcols) {
#pragma unroll
              for (int j = 0; j < 16; j += 4)
                *reinterpret_cast<float4 *>(zr + c + j) = make_float4(z[j], z[j + 1], z[j + 2], z[j + 3]);
            } else {
#pragma unroll
              for (int j = 0; j < 16; ++j)
                if (c + j < p.zcols) zr[c + j] = z[j];
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&tempty[a]));
        continue;
      }
      if (p.wide) {
        // x.c = (column j) + (column BN + j)
        for (int c = 0; c < p.BN; c += 16) {
          tmem_ld16(taddr + (uint32_t)c, ra);
          tmem_ld16(taddr + (uint32_t)(p.BN + c), rb);
          tmem_ld_wait(ra);
          tmem_ld_wait(rb);
#pragma unroll
          for (int j = 0; j < 16; ++j) ra[j] = __float_as_uint(__uint_as_float(ra[j]) + __uint_as_float(rb[j]));
          epilogue_group(ra, cb + c, c, best1, best2, best3, idx1, idx2);
        }
      } else {
        tmem_ld16(taddr, ra);
        tmem_ld_wait(ra);
        for (int c = 0; c < p.BN; c += 32) {
          const bool more1 = c + 16 < p.BN, more2 = c + 32 < p.BN;
          if (more1) tmem_ld16(taddr + (uint32_t)(c + 16), rb);
          epilogue_group(ra, cb + c, c, best1, best2, best3, idx1, idx2);
          if (more1) {
            tmem_ld_wait(rb);
            if (more2) tmem_ld16(taddr + (uint32_t)(c + 32), ra);
            epilogue_group(rb, cb + c + 16, c + 16, best1, best2, best3, idx1, idx2);
            if (more2) tmem_ld_wait(ra);
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&tempty[a]));
      const int64_t row = (int64_t)tile * kBM + r;
      if (row < p.N) obj += finish_row<false>(p, row, xr, best1, best2, best3, idx1, idx2, cn_max, sqrt_cn_max);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) obj += __shfl_xor_sync(0xffffffffu, obj, o);
    if (lane == 0 && obj != 0.0) atomicAdd(&p.hdr->objective, obj);
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, p.tmem_cols);
  }
}

// Exact re-score of near-tie rows: direct fp32 differences, squared and summed
// per lane in fp32 (a sum of non-negative terms), combined across the warp;
// ties to the lowest k.  A queued row names its two candidates (best and
// runner-up of the tensor-core pass), or -1 for "compare all K" when a third
// centre was also within the margin.
// Row segment loads: VW consecutive elements (16 bytes when vectorised).
template <int DT, int VW>
__device__ __forceinline__ void load_x(const void *Xv, int64_t off, float (&v)[VW]) {
  if constexpr (DT == HME_F32) {
    const float *p = reinterpret_cast<const float *>(Xv) + off;
    if constexpr (VW == 4) {
      const float4 f = __ldg(reinterpret_cast<const float4 *>(p));
      v[0] = f.x, v[1] = f.y, v[2] = f.z, v[3] = f.w;
    } else {
#pragma unroll
      for (int e = 0; e < VW; ++e) v[e] = __ldg(p + e);
    }
  } else {
    const __nv_bfloat16 *p = reinterpret_cast<const __nv_bfloat16 *>(Xv) + off;
    if constexpr (VW == 8) {
      const uint4 u = __ldg(reinterpret_cast<const uint4 *>(p));
      const __nv_bfloat162 *h = reinterpret_cast<const __nv_bfloat162 *>(&u);
#pragma unroll
      for (int t = 0; t < VW / 2; ++t) {
        const float2 f = __bfloat1622float2(h[t]);
        v[2 * t] = f.x, v[2 * t + 1] = f.y;
      }
    } else {
#pragma unroll
      for (int e = 0; e < VW; ++e) v[e] = __bfloat162float(p[e]);
    }
  }
}

// Centre values the assign step compares against (bf16-rounded for bf16 features).
template <int DT, int VW>
__device__ __forceinline__ void load_c(const float *C, int64_t off, float (&v)[VW]) {
  if constexpr (VW % 4 == 0) {
#pragma unroll
    for (int q = 0; q < VW / 4; ++q) {
      const float4 f = __ldg(reinterpret_cast<const float4 *>(C + off) + q);
      v[4 * q] = f.x, v[4 * q + 1] = f.y, v[4 * q + 2] = f.z, v[4 * q + 3] = f.w;
    }
  } else {
#pragma unroll
    for (int e = 0; e < VW; ++e) v[e] = __ldg(C + off + e);
  }
  if constexpr (DT == HME_BF16) {
#pragma unroll
    for (int e = 0; e < VW; ++e) v[e] = __bfloat162float(__float2bfloat16_rn(v[e]));
  }
}

__device__ __forceinline__ float warp_sum_f(float s) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  return s;
}


// Exact re-score of near-tie rows with two candidates: one warp per row, one
// pass over the row computing both sums of squared differences (fp32 per lane,
// a sum of non-negative terms, then across the warp); ties to the lower index.
template <int DT, int VW>
__global__ void __launch_bounds__(256) rescore_pair_kernel(const void *__restrict__ Xv, int d, int64_t ldx,
                                                           const float *__restrict__ C, int32_t *labels, float *mind,
                                                           Header *hdr, const int32_t *__restrict__ flagged,
                                                           unsigned long long *full_keys_end) {
  const int lane = threadIdx.x & 31;
  const int gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int nw = (gridDim.x * blockDim.x) >> 5;
  const uint32_t count = *((volatile uint32_t *)&hdr->rescore_count);
  if (full_keys_end) {  // the all-K re-score that follows merges into these keys
    const uint32_t nfull = *((volatile uint32_t *)&hdr->rescore_full_count);
    for (uint32_t f = blockIdx.x * blockDim.x + threadIdx.x; f < nfull; f += gridDim.x * blockDim.x)
      full_keys_end[-1 - (int64_t)f] = ~0ull;
  }
  double obj = 0.0;
  for (uint32_t f = gw; f < count; f += nw) {
    const int64_t row = flagged[3 * f + 0];
    const int i1 = flagged[3 * f + 1];
    const int i2 = flagged[3 * f + 2];
    float s1 = 0.0f, s2 = 0.0f;
#pragma unroll 4
    for (int j = lane * VW; j < d; j += 32 * VW) {
      float x[VW], c1[VW], c2[VW];
      load_x<DT, VW>(Xv, row * ldx + j, x);
      load_c<DT, VW>(C, (int64_t)i1 * d + j, c1);
      load_c<DT, VW>(C, (int64_t)i2 * d + j, c2);
#pragma unroll
      for (int e = 0; e < VW; ++e) {
        const float t1 = x[e] - c1[e], t2 = x[e] - c2[e];
        s1 = fmaf(t1, t1, s1);
        s2 = fmaf(t2, t2, s2);
      }
    }
    s1 = warp_sum_f(s1);
    s2 = warp_sum_f(s2);
    const bool first = s1 < s2 || (s1 == s2 && i1 < i2);
    if (lane == 0) {
      labels[row] = first ? i1 : i2;
      if (mind) mind[row] = first ? s1 : s2;
      obj += (double)(first ? s1 : s2);
    }
  }
  if (lane == 0 && obj != 0.0) atomicAdd(&hdr->objective, obj);
}

// Exact re-score against all K centres when K is small (one N-chunk): one block
// per queued row; the row is cached in shared memory and the 8 warps split the
// centres, each lane summing (x_j - c_j)^2 over its strided elements in fp32
// (16-byte loads of c), then across the warp and across the warps; ties to the
// lowest index.  Each warp streams kRowKB centre rows at a time, so the
// latency is about K / (8 kRowKB) passes over one centre row.
constexpr int kRowKB = 4;

template <int DT, int VW>
__global__ void __launch_bounds__(256) rescore_row_kernel(const void *__restrict__ Xv, int d, int64_t ldx,
                                                          const float *__restrict__ C, int K, int32_t *labels,
                                                          float *mind, Header *hdr,
                                                          const int32_t *__restrict__ full_rows) {
  extern __shared__ float xrow[];
  __shared__ float wv[8];
  __shared__ int wk[8];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint32_t count = *((volatile uint32_t *)&hdr->rescore_full_count);
  double obj = 0.0;
  for (uint32_t f = blockIdx.x; f < count; f += gridDim.x) {
    const int64_t row = full_rows[f];
    for (int j = threadIdx.x; j < d; j += blockDim.x) {
      float x;
      if (DT == HME_BF16)
        x = __bfloat162float(reinterpret_cast<const __nv_bfloat16 *>(Xv)[row * ldx + j]);
      else
        x = reinterpret_cast<const float *>(Xv)[row * ldx + j];
      xrow[j] = x;
    }
    __syncthreads();
    float bv = INFINITY;
    int bk = 0x7fffffff;
    // each warp takes kRowKB centres at a time (their loads in flight together);
    // k ascends within a warp
    for (int k0 = warp * kRowKB; k0 < K; k0 += 8 * kRowKB) {
      float sacc[kRowKB];
#pragma unroll
      for (int b = 0; b < kRowKB; ++b) sacc[b] = 0.0f;
#pragma unroll 2
      for (int j = lane * VW; j < d; j += 32 * VW) {
#pragma unroll
        for (int b = 0; b < kRowKB; ++b) {
          float c[VW];  // centres past K repeat the last one; their sums are discarded
          load_c<DT, VW>(C, (int64_t)min(k0 + b, K - 1) * d + j, c);
#pragma unroll
          for (int e = 0; e < VW; ++e) {
            const float t = xrow[j + e] - c[e];
            sacc[b] = fmaf(t, t, sacc[b]);
          }
        }
      }
#pragma unroll
      for (int b = 0; b < kRowKB; ++b) {
        const float v = warp_sum_f(sacc[b]);
        if (k0 + b < K && v < bv) {
          bv = v;
          bk = k0 + b;
        }
      }
    }
    if (lane == 0) {
      wv[warp] = bv;
      wk[warp] = bk;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      float v = wv[0];
      int kk = wk[0];
      for (int w = 1; w < 8; ++w)
        if (wv[w] < v || (wv[w] == v && wk[w] < kk)) {
          v = wv[w];
          kk = wk[w];
        }
      labels[row] = kk;
      if (mind) mind[row] = v;
      obj += (double)v;
    }
    __syncthreads();
  }
  if (threadIdx.x == 0 && obj != 0.0) atomicAdd(&hdr->objective, obj);
}

// Exact re-score of near-tie rows against all K centres: a small tiled
// "distance GEMM" on the CUDA cores.  A work item is 16 x RPT queued rows and
// one slice of the centres, walked 64 centres and 32 dimensions at a time
// through shared memory (rows row-major; centres dimension-major, so that a
// thread reads its four centres with one 16-byte load; with CV the centres
// come from global memory in 16-byte loads with the lanes along the centres,
// so that the transposing stores hit distinct banks).  Thread (ty, tx) of a
// 16 x 16 grid owns rows ty + 16i (i < RPT) and centres 4tx .. 4tx+3: 4 RPT
// distances for RPT + 1 shared loads per dimension.  RPT is 4 (64-row items)
// or 2 (32-row items, twice as many), whichever is estimated to finish first:
// a long queue runs faster in the larger tile, a short one (a small routed
// batch) in more, smaller items.  sum_j (x_j - c_j)^2 is formed in fp32 per
// 32-wide chunk (j ascending) and the chunk sums are added in fp32 in chunk
// order, whatever RPT (relative error below (32 + d/32) 2^-24, all terms
// non-negative).  With many queued rows a slice is all K centres; with few the
// centres are split over the blocks so that the work still spreads over the
// GPU.  A slice's best (distance, centre) per row is merged with a 64-bit
// atomicMin on (distance bits << 32 | centre): the distances are non-negative,
// so their bit patterns order like the values, and equal distances keep the
// lower centre.  rescore_full_finish_kernel then writes labels, distances and
// the objective.
//
// The keys of queued row f sit at full_keys_end[-1 - f]: the 8-byte aligned
// tail of the pair queue (3 words per row of the call).  Rows queued for a
// pair (3 words each) and for all K (2 words each) number at most N together,
// so 3 pairs + 2 full <= 3N - full <= 3N - 1 words: the keys never reach a
// queued pair.
constexpr int kFRmax = 64, kFC = 64, kFD = 32;

struct FullTiles {
  float (*xs)[kFD + 1];   // [kFRmax][kFD + 1] rows
  float (*cs)[kFC + 4];   // [kFD][kFC + 4] centres, dimension-major
  float *best_v;          // [kFRmax]
  int *best_k;            // [kFRmax]
  int64_t *rows;          // [kFRmax]
};

template <int DT, bool CV, int RPT>
__device__ __forceinline__ void rescore_full_body(const void *__restrict__ Xv, int d, int64_t ldx,
                                                  const float *__restrict__ C, int K, uint32_t count,
                                                  const int32_t *__restrict__ full_rows,
                                                  unsigned long long *full_keys_end, const FullTiles &sm) {
  constexpr int kFR = 16 * RPT;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  const uint32_t ntiles = (count + kFR - 1) / kFR;
  const int kt = (K + kFC - 1) / kFC;  // tiles of kFC centres
  const int ks = (int)min((uint32_t)kt, max(1u, gridDim.x / max(ntiles, 1u)));  // slices per row tile
  const uint32_t items = ntiles * (uint32_t)ks;
  for (uint32_t it = blockIdx.x; it < items; it += gridDim.x) {
    const uint32_t b0 = (it / (uint32_t)ks) * kFR;
    const int sl = (int)(it % (uint32_t)ks);
    const int kbeg = (sl * kt / ks) * kFC, kend = min(K, ((sl + 1) * kt / ks) * kFC);
    const int nr = (int)min((uint32_t)kFR, count - b0);
    if (threadIdx.x < kFR) {
      sm.rows[threadIdx.x] = threadIdx.x < nr ? (int64_t)full_rows[b0 + threadIdx.x] : -1;
      sm.best_v[threadIdx.x] = INFINITY;
      sm.best_k[threadIdx.x] = 0;
    }
    __syncthreads();
    for (int k0 = kbeg; k0 < kend; k0 += kFC) {
      float tot[RPT][4];
#pragma unroll
      for (int i = 0; i < RPT; ++i)
#pragma unroll
        for (int q = 0; q < 4; ++q) tot[i][q] = 0.0f;
      for (int j0 = 0; j0 < d; j0 += kFD) {
        for (int e = threadIdx.x; e < kFR * kFD; e += 256) {
          const int r = e / kFD, j = e - r * kFD;
          const int64_t row = sm.rows[r];
          float x = 0.0f;
          if (row >= 0 && j0 + j < d) {
            if (DT == HME_BF16)
              x = __bfloat162float(reinterpret_cast<const __nv_bfloat16 *>(Xv)[row * ldx + j0 + j]);
            else
              x = reinterpret_cast<const float *>(Xv)[row * ldx + j0 + j];
          }
          sm.xs[r][j] = x;
        }
        if (CV) {  // 16-byte loads, lanes along the centres: conflict-free stores
          for (int e = threadIdx.x; e < kFC * kFD / 4; e += 256) {
            const int c = e % kFC, jq = 4 * (e / kFC);
            const int k = k0 + c;
            float4 v = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
            if (k < K && j0 + jq < d) {  // d % 4 == 0: the whole vector is inside the row
              v = __ldg(reinterpret_cast<const float4 *>(C + (int64_t)k * d + j0 + jq));
              if (DT == HME_BF16) {
                v.x = __bfloat162float(__float2bfloat16_rn(v.x));
                v.y = __bfloat162float(__float2bfloat16_rn(v.y));
                v.z = __bfloat162float(__float2bfloat16_rn(v.z));
                v.w = __bfloat162float(__float2bfloat16_rn(v.w));
              }
            }
            sm.cs[jq][c] = v.x;
            sm.cs[jq + 1][c] = v.y;
            sm.cs[jq + 2][c] = v.z;
            sm.cs[jq + 3][c] = v.w;
          }
        } else {
          for (int e = threadIdx.x; e < kFC * kFD; e += 256) {
            const int c = e / kFD, j = e - c * kFD;
            const int k = k0 + c;
            float v = 0.0f;
            if (k < K && j0 + j < d) {
              v = __ldg(C + (int64_t)k * d + j0 + j);
              if (DT == HME_BF16) v = __bfloat162float(__float2bfloat16_rn(v));
            }
            sm.cs[j][c] = v;
          }
        }
        __syncthreads();
        float part[RPT][4];
#pragma unroll
        for (int i = 0; i < RPT; ++i)
#pragma unroll
          for (int q = 0; q < 4; ++q) part[i][q] = 0.0f;
#pragma unroll 4
        for (int j = 0; j < kFD; ++j) {
          float x[RPT];
#pragma unroll
          for (int i = 0; i < RPT; ++i) x[i] = sm.xs[ty + 16 * i][j];
          const float4 c4 = *reinterpret_cast<const float4 *>(&sm.cs[j][4 * tx]);
          const float c[4] = {c4.x, c4.y, c4.z, c4.w};
#pragma unroll
          for (int i = 0; i < RPT; ++i)
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const float t = x[i] - c[q];
              part[i][q] = fmaf(t, t, part[i][q]);
            }
        }
#pragma unroll
        for (int i = 0; i < RPT; ++i)
#pragma unroll
          for (int q = 0; q < 4; ++q) tot[i][q] += part[i][q];
        __syncthreads();
      }
#pragma unroll
      for (int i = 0; i < RPT; ++i) {
        float v = INFINITY;
        int kk = 0x7fffffff;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int k = k0 + 4 * tx + q;
          if (k < K && tot[i][q] < v) {
            v = tot[i][q];
            kk = k;
          }
        }
#pragma unroll
        for (int o = 8; o > 0; o >>= 1) {  // the 16 threads of one ty share a half-warp
          const float ov = __shfl_xor_sync(0xffffffffu, v, o);
          const int ok = __shfl_xor_sync(0xffffffffu, kk, o);
          if (ov < v || (ov == v && ok < kk)) {
            v = ov;
            kk = ok;
          }
        }
        const int rl = ty + 16 * i;
        if (tx == 0 && (v < sm.best_v[rl] || (v == sm.best_v[rl] && kk < sm.best_k[rl]))) {
          sm.best_v[rl] = v;
          sm.best_k[rl] = kk;
        }
      }
    }
    __syncthreads();
    if (threadIdx.x < nr) {
      const unsigned long long key =
          ((unsigned long long)__float_as_uint(sm.best_v[threadIdx.x]) << 32) | (uint32_t)sm.best_k[threadIdx.x];
      atomicMin(&full_keys_end[-1 - (int64_t)(b0 + threadIdx.x)], key);
    }
    __syncthreads();
  }
}

template <int DT, bool CV>
__global__ void __launch_bounds__(256) rescore_full_kernel(const void *__restrict__ Xv, int d, int64_t ldx,
                                                           const float *__restrict__ C, int K, const Header *hdr,
                                                           const int32_t *__restrict__ full_rows,
                                                           unsigned long long *full_keys_end) {
  __shared__ float xs[kFRmax][kFD + 1];
  __shared__ __align__(16) float cs[kFD][kFC + 4];
  __shared__ float best_v[kFRmax];
  __shared__ int best_k[kFRmax];
  __shared__ int64_t rows[kFRmax];
  const FullTiles sm{xs, cs, best_v, best_k, rows};
  const uint32_t count = *((volatile const uint32_t *)&hdr->rescore_full_count);
  // Estimated time (x gridDim) with each row tile: the larger of its longest
  // work item and all its work spread over the blocks; a 64-row tile costs
  // 1.6x a 32-row one (measured: 16 against 10).
  const uint64_t kt = (uint64_t)((K + kFC - 1) / kFC), g = gridDim.x;
  auto est = [&](uint64_t fr, uint64_t cost) -> uint64_t {
    const uint64_t nt = (count + fr - 1) / fr;
    const uint64_t ks = min(kt, max((uint64_t)1, g / max(nt, (uint64_t)1)));
    return max((kt + ks - 1) / ks * cost * g, nt * kt * cost);
  };
  if (est(64, 16) < est(32, 10))
    rescore_full_body<DT, CV, 4>(Xv, d, ldx, C, K, count, full_rows, full_keys_end, sm);
  else
    rescore_full_body<DT, CV, 2>(Xv, d, ldx, C, K, count, full_rows, full_keys_end, sm);
}

// The all-K re-score's result per queued row: label, distance, objective.
__global__ void __launch_bounds__(256) rescore_full_finish_kernel(int32_t *labels, float *mind, Header *hdr,
                                                                  const int32_t *__restrict__ full_rows,
                                                                  const unsigned long long *full_keys_end) {
  const uint32_t count = *((volatile uint32_t *)&hdr->rescore_full_count);
  double obj = 0.0;
  for (uint32_t f = blockIdx.x * blockDim.x + threadIdx.x; f < count; f += gridDim.x * blockDim.x) {
    const unsigned long long key = full_keys_end[-1 - (int64_t)f];
    const int64_t row = full_rows[f];
    const float v = __uint_as_float((uint32_t)(key >> 32));
    labels[row] = (int32_t)(uint32_t)(key & 0xffffffffu);
    if (mind) mind[row] = v;
    obj += (double)v;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) obj += __shfl_xor_sync(0xffffffffu, obj, o);
  if ((threadIdx.x & 31) == 0 && obj != 0.0) atomicAdd(&hdr->objective, obj);
}

// ---------------------------------------------------------------------------
// host side: tensor maps and launch
// ---------------------------------------------------------------------------
typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn get_encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(f);
  });
  return fn;
}

// bf16 matrix rows x cols (row stride ld elements), box = box_rows x 64 columns, 128-byte swizzle.
int make_map(CUtensorMap *m, const void *ptr, uint64_t rows, uint64_t cols, uint64_t ld, uint32_t box_rows) {
  EncodeTiledFn enc = get_encode_fn();
  if (!enc) return fail(HME_ECUDA, "cuTensorMapEncodeTiled is not available from the driver");
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {ld * 2};
  cuuint32_t box[2] = {(cuuint32_t)kBK, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS)
    return fail(HME_ECUDA, "cuTensorMapEncodeTiled failed (%d) for %llu x %llu, ld %llu", (int)r,
                (unsigned long long)rows, (unsigned long long)cols, (unsigned long long)ld);
  return HME_OK;
}

// fp32 matrix rows x cols (row stride ld elements), box = box_rows rows x 32
// columns (128 bytes), 128-byte swizzle.
int make_map_f32(CUtensorMap *m, const void *ptr, uint64_t rows, uint64_t cols, uint64_t ld,
                 uint32_t box_rows = kBM) {
  EncodeTiledFn enc = get_encode_fn();
  if (!enc) return fail(HME_ECUDA, "cuTensorMapEncodeTiled is not available from the driver");
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {ld * 4};
  cuuint32_t box[2] = {32, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void *>(ptr), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS)
    return fail(HME_ECUDA, "cuTensorMapEncodeTiled (fp32) failed (%d) for %llu x %llu, ld %llu", (int)r,
                (unsigned long long)rows, (unsigned long long)cols, (unsigned long long)ld);
  return HME_OK;
}

}  // namespace

int make_bf16_map(CUtensorMap *m, const void *ptr, uint64_t rows, uint64_t cols, uint64_t ld, uint32_t box_rows) {
  return make_map(m, ptr, rows, cols, ld, box_rows);
}

// Epilogue warps per lane quarter of the resident-row kernel.  On 8e6 rows of
// the 5e7 x 256, K = 4096 set, with the lean MMA issue loop: four 12.58 ms,
// two 12.84 ms (when the MMA thread still spent many instructions per MMA,
// two had been the fastest: the epilogue warps sharing its sub-partition
// took its issue slots).
constexpr int kAresCS = 4;

int launch_assign(const void *Xa, const void *Xb, int64_t N, int64_t lda, const AssignGeom &g, const void *chi,
                  const __nv_bfloat16 *clo, const float *cn, const float *xn, int32_t *labels, float *mind,
                  Header *hdr, int32_t *flagged, int32_t *full_rows, float4 *part, cudaStream_t s) {
  if (N == 0) return HME_OK;
  CUtensorMap mA0, mA1, mB0, mB1;
  int rc;
  if (g.tf32) {  // fp32 rows and tf32-rounded fp32 centres, 32-column boxes
    if ((rc = make_map_f32(&mA0, Xa, (uint64_t)N, (uint64_t)g.d, (uint64_t)lda, kBM)) != HME_OK) return rc;
    if ((rc = make_map_f32(&mB0, chi, (uint64_t)g.K, (uint64_t)g.d, (uint64_t)g.ldc, (uint32_t)g.BN)) != HME_OK)
      return rc;
  } else {
    if ((rc = make_map(&mA0, Xa, (uint64_t)N, (uint64_t)g.d, (uint64_t)lda, kBM)) != HME_OK) return rc;
    if ((rc = make_map(&mB0, chi, (uint64_t)g.K, (uint64_t)g.d, (uint64_t)g.ldp, (uint32_t)g.BN)) != HME_OK)
      return rc;
  }
  if (g.nprod == 3) {
    if ((rc = make_map(&mA1, Xb, (uint64_t)N, (uint64_t)g.d, (uint64_t)lda, kBM)) != HME_OK) return rc;
    if ((rc = make_map(&mB1, clo, (uint64_t)g.K, (uint64_t)g.d, (uint64_t)g.ldp, (uint32_t)g.BN)) != HME_OK)
      return rc;
  } else {
    mA1 = mA0;
    mB1 = mB0;
  }
  AssignParams p;
  p.N = N;
  p.num_kb = (g.d + g.kblk - 1) / g.kblk;
  p.BN = g.BN;
  p.nchunks = g.nchunks;
  p.num_tiles = (int)((N + kBM * g.mt - 1) / (kBM * g.mt));
  p.a_bytes = kBM * kBK * 2;
  p.b_bytes = (uint32_t)g.BN * kBK * 2;
  const int nops = g.nprod == 3 ? 2 : 1;
  p.a_res_bytes = g.ares ? (uint32_t)(g.mt * p.num_kb * nops) * p.a_bytes : 0u;
  p.stage_bytes = nops * ((g.ares ? 0u : (uint32_t)g.mt * p.a_bytes) + p.b_bytes);
  // epilogue warps per (row tile, lane quarter): two for bf16 features, whose
  // one product per k-step leaves the epilogue scan as the longer pipeline
  const int cs = g.nprod == 3 ? 1 : (g.ares ? kAresCS : 2);
  const size_t ctrl_bytes = 512 + (size_t)4 * g.mt * kMaxBN * sizeof(float) +
                            (size_t)2 * 4 * g.mt * (cs - 1) * 32 * sizeof(float4);
  const size_t budget = 227 * 1024 - 1024 - ctrl_bytes - p.a_res_bytes;
  int stages = (int)(budget / p.stage_bytes);
  if (stages > 8) stages = 8;
  if (stages < 2) return fail(HME_EINTERNAL, "assign: stage of %u bytes does not fit twice", p.stage_bytes);
  p.stages = stages;
  p.nbuf = g.nbuf;
  uint32_t stride = 32;
  while (stride < (uint32_t)(g.mt * g.BN)) stride <<= 1;
  p.acc_stride = stride;
  p.tmem_cols = (uint32_t)g.nbuf * stride;
  if (p.tmem_cols > 512) return fail(HME_EINTERNAL, "assign: %u TMEM columns", p.tmem_cols);
  p.xn = xn;
  p.cn = cn;
  p.labels = labels;
  p.mind = mind;
  p.hdr = hdr;
  p.flagged = flagged;
  p.full_rows = full_rows;
  p.limit_ns = wait_limit_ns();
  // accumulation steps along d: 16 elements per bf16 MMA step, 8 per tf32 step
  const int steps = g.tf32 ? (g.d + 7) / 8 : (g.d + 15) / 16;
  p.err_acc = (float)((double)steps * g.nprod * 0x1p-22 + 0x1p-20);
  p.err_split = g.nprod == 3 ? 0x1p-14f : 0.0f;
  // split operands: the dropped xl.cl; tf32 operands: their rounding (6.002 * 2^-10)
  p.err_ll = g.nprod == 3 ? 0x1.1p-14f : (g.tf32 ? (float)(6.002 * 0x1p-10) : 0.0f);
  const size_t smem = (size_t)p.a_res_bytes + (size_t)stages * p.stage_bytes + 1024 + ctrl_bytes;
  const bool lean = g.nchunks > 1;
  // Few row tiles (a small routed batch) would leave most SMs idle: spread
  // each tile's N-chunks over up to kMaxSlices CTAs (lean scan only).
  p.slices = 1;
  p.cps = g.nchunks;
  p.part = nullptr;
  if (lean && !g.tf32 && part && N <= kSplitRows && 2 * p.num_tiles <= num_sms()) {
    int sl = num_sms() / p.num_tiles;
    if (sl > g.nchunks) sl = g.nchunks;
    if (sl > kMaxSlices) sl = kMaxSlices;
    if (sl >= 2) {
      p.cps = (g.nchunks + sl - 1) / sl;
      p.slices = (g.nchunks + p.cps - 1) / p.cps;  // no empty slice
      p.part = part;
    }
  }
  int grid = num_sms();
  if (grid > p.num_tiles * p.slices) grid = p.num_tiles * p.slices;
  cudaError_t e;
  using Kern = void (*)(const CUtensorMap, const CUtensorMap, const CUtensorMap, const CUtensorMap, const AssignParams);
  Kern kern;
  // Several N-chunks of the three-product split: the top-three scan, so that
  // near ties with two candidates are re-scored on those two (the split is
  // bound by its MMAs, and the wider scan cuts the all-K re-scores about a
  // hundredfold: 1.6e7 x 512, K = 1024 features, 8.8 -> 7.6 ms for 4e6 rows).
  // bf16 features keep the lean scan: their kernel is bound by the epilogue,
  // where the top-three scan cost half as much again (5e7 x 256, K = 4096
  // features: 14.2 -> 21.3 ms for 8e6 rows) as the all-K re-scores it saves.
  // Centre slices always use the lean states the merge kernel combines.
  const bool top3 = lean && p.slices == 1 && g.nprod == 3;
  if (g.tf32)
    kern = assign_kernel<1, false, 2, false, 2, true>;  // top-three scan: two-candidate near ties re-scored cheaply
  else if (g.nprod == 3)
    kern = top3 ? assign_kernel<3, false, 1, false, 1, false, true>
                : (lean ? assign_kernel<3, true, 1, false, 1> : assign_kernel<3, false, 1, false, 1>);
  else if (g.ares)
    kern = assign_kernel<1, true, 1, true, kAresCS>;
  else
    kern = lean ? assign_kernel<1, true, 2, false, 2> : assign_kernel<1, false, 2, false, 2>;
  e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return cuda_fail(e, "assign: set smem");
  kern<<<grid, 64 + 128 * g.mt * cs, smem, s>>>(mA0, mA1, mB0, mB1, p);
  count_launch();
  if (p.slices > 1) {
    assign_merge_kernel<<<(unsigned)((N + kMergeRows - 1) / kMergeRows), 256, 0, s>>>(p);
    count_launch();
  }
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "assign kernel launch");
  return HME_OK;
}

bool split_eligible(const void *X, int64_t ldx, const AssignGeom &g) {
  return g.nprod == 3 && g.nchunks == 1 && (reinterpret_cast<uintptr_t>(X) & 15u) == 0 && ldx % 4 == 0;
}

int launch_assign_split(const float *X, int64_t N, int64_t ldx, const AssignGeom &g, const __nv_bfloat16 *chi,
                        const __nv_bfloat16 *clo, const float *cn, int32_t *labels, float *mind, Header *hdr,
                        int32_t *flagged, int32_t *full_rows, const SplitOut &out, cudaStream_t s) {
  __nv_bfloat16 *xhi_out = out.xhi, *xlo_out = out.xlo;
  float *xn_out = out.xn;
  if (N == 0) return HME_OK;
  CUtensorMap mX, mB0, mB1, mOh, mOl;
  int rc;
  if ((rc = make_map_f32(&mX, X, (uint64_t)N, (uint64_t)g.d, (uint64_t)ldx)) != HME_OK) return rc;
  if (xhi_out) {  // 64 columns x 32 rows: one converter warp's share of a k-block
    if ((rc = make_map(&mOh, xhi_out, (uint64_t)N, (uint64_t)g.d, (uint64_t)g.ldp, 32)) != HME_OK) return rc;
    if ((rc = make_map(&mOl, xlo_out, (uint64_t)N, (uint64_t)g.d, (uint64_t)g.ldp, 32)) != HME_OK) return rc;
  }
  if ((rc = make_map(&mB0, chi, (uint64_t)g.K, (uint64_t)g.d, (uint64_t)g.ldp, (uint32_t)g.BN)) != HME_OK)
    return rc;
  if ((rc = make_map(&mB1, clo, (uint64_t)g.K, (uint64_t)g.d, (uint64_t)g.ldp, (uint32_t)g.BN)) != HME_OK)
    return rc;
  AssignParams p{};
  p.N = N;
  p.num_kb = (g.d + kBK - 1) / kBK;
  p.BN = g.BN;
  p.nchunks = 1;
  p.slices = 1;
  p.cps = 1;
  p.write_split = xhi_out ? 1 : 0;
  p.xn_out = xn_out;
  p.z_out = out.z;
  p.ldz = out.ldz;
  p.zcols = out.zcols;
  p.zvec = out.z && (reinterpret_cast<uintptr_t>(out.z) & 15u) == 0 && out.ldz % 4 == 0;
  p.num_tiles = (int)((N + kBM - 1) / kBM);
  p.a_bytes = 0;
  p.b_bytes = (uint32_t)g.BN * kBK * 2;
  p.b_stage_bytes = 2 * p.b_bytes;
  p.a_res_bytes = 0;
  // TMEM: accumulators (double-buffered when they fit) + 4 split A stages of 64 columns
  p.wide = 2 * g.BN <= kMaxBN ? 1 : 0;
  uint32_t stride = 32;
  while (stride < (uint32_t)(p.wide ? 2 * g.BN : g.BN)) stride <<= 1;
  p.acc_stride = stride;
  p.nbuf = (2 * stride + 64u * 4u <= 512u) ? 2 : 1;
  p.a_col0 = (uint32_t)p.nbuf * stride;
  p.st_stages = 4;
  p.tmem_cols = 512;
  if (p.a_col0 + 64u * p.st_stages > 512u) return fail(HME_EINTERNAL, "assign (split): TMEM columns");
  // shared memory: fp32 stages get what the centre stages leave
  const size_t ctrl_bytes = 512 + (size_t)4 * kBM * sizeof(float) + (size_t)4 * kMaxBN * sizeof(float);
  const size_t budget = 227 * 1024 - 1024 - ctrl_bytes;
  // Both rings hide a load latency per k-block (HBM for the rows, L2 for the
  // centres, which queues behind the same traffic): four fp32 stages, then as
  // many centre stages as fit (at most five, at least two).
  int sx = 4;
  int sb = (int)((budget - (size_t)sx * kXStage) / p.b_stage_bytes);
  if (sb > 5) sb = 5;
  while (sb < 2 && sx > 2) {
    --sx;
    sb = (int)((budget - (size_t)sx * kXStage) / p.b_stage_bytes);
    if (sb > 5) sb = 5;
  }
  if (sb < 2) return fail(HME_EINTERNAL, "assign (split): a centre stage of %u bytes does not fit", p.b_stage_bytes);
  p.sb_stages = sb;
  p.stages = sx;
  p.xn = nullptr;
  p.cn = cn;
  p.labels = labels;
  p.mind = mind;
  p.hdr = hdr;
  p.flagged = flagged;
  p.full_rows = full_rows;
  p.limit_ns = wait_limit_ns();
  p.err_acc = (float)((double)((g.d + 15) / 16) * g.nprod * 0x1p-22 + 0x1p-20);
  p.err_split = 0x1p-14f;
  p.err_ll = 0x1.1p-14f;
  const size_t smem = 1024 + (size_t)sx * kXStage + (size_t)p.sb_stages * p.b_stage_bytes + ctrl_bytes;
  int grid = num_sms();
  if (grid > p.num_tiles) grid = p.num_tiles;
  cudaError_t e = cudaFuncSetAttribute(assign_split_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return cuda_fail(e, "assign (split): set smem");
  assign_split_kernel<<<grid, kSplitThreads, smem, s>>>(mX, mB0, mB1, xhi_out ? mOh : mB0, xhi_out ? mOl : mB1, p);
  count_launch();
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "assign (split) kernel launch");
  return HME_OK;
}

cudaError_t launch_rescore(const void *X, int64_t N, int d, int64_t ldx, int dtype, const float *C, int K,
                           int32_t *labels, float *mind, Header *hdr, int32_t *flagged,
                           const int32_t *full_rows, cudaStream_t s) {
  if (N == 0) return cudaSuccess;
  const int grid = num_sms() * 4;
  // the queues hold at most N rows: a warp per queued pair, a thread per finished row
  const int gpair = (int)std::min<int64_t>(grid, (N + 7) / 8);
  const int gfin = (int)std::min<int64_t>(grid, (N + 255) / 256);
  const bool al = ((reinterpret_cast<uintptr_t>(X) | reinterpret_cast<uintptr_t>(C)) & 15u) == 0;
  // all-K rows: block per row for few centres (low latency), tiled otherwise
  const bool row_path = K <= 128;
  const bool cvec = (reinterpret_cast<uintptr_t>(C) & 15u) == 0 && d % 4 == 0;
  const size_t row_smem = (size_t)d * sizeof(float);
  // keys of the all-K re-score: the 8-byte aligned tail of the pair queue (3N words)
  unsigned long long *keys_end =
      row_path ? nullptr : reinterpret_cast<unsigned long long *>(flagged + ((3 * N) & ~(int64_t)1));
  if (row_path && row_smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(dtype == HME_BF16 ? rescore_row_kernel<HME_BF16, 1>
                                                           : (cvec ? rescore_row_kernel<HME_F32, 4>
                                                                   : rescore_row_kernel<HME_F32, 1>),
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)row_smem);
    if (e != cudaSuccess) return e;
  }
  if (dtype == HME_BF16) {
    if (al && d % 8 == 0 && ldx % 8 == 0)
      rescore_pair_kernel<HME_BF16, 8><<<gpair, 256, 0, s>>>(X, d, ldx, C, labels, mind, hdr, flagged, keys_end);
    else
      rescore_pair_kernel<HME_BF16, 1><<<gpair, 256, 0, s>>>(X, d, ldx, C, labels, mind, hdr, flagged, keys_end);
    if (row_path)
      rescore_row_kernel<HME_BF16, 1><<<grid, 256, row_smem, s>>>(X, d, ldx, C, K, labels, mind, hdr, full_rows);
    else if (cvec)
      rescore_full_kernel<HME_BF16, true><<<grid, 256, 0, s>>>(X, d, ldx, C, K, hdr, full_rows, keys_end);
    else
      rescore_full_kernel<HME_BF16, false><<<grid, 256, 0, s>>>(X, d, ldx, C, K, hdr, full_rows, keys_end);
  } else {
    if (al && d % 4 == 0 && ldx % 4 == 0)
      rescore_pair_kernel<HME_F32, 4><<<gpair, 256, 0, s>>>(X, d, ldx, C, labels, mind, hdr, flagged, keys_end);
    else
      rescore_pair_kernel<HME_F32, 1><<<gpair, 256, 0, s>>>(X, d, ldx, C, labels, mind, hdr, flagged, keys_end);
    if (row_path && cvec)
      rescore_row_kernel<HME_F32, 4><<<grid, 256, row_smem, s>>>(X, d, ldx, C, K, labels, mind, hdr, full_rows);
    else if (row_path)
      rescore_row_kernel<HME_F32, 1><<<grid, 256, row_smem, s>>>(X, d, ldx, C, K, labels, mind, hdr, full_rows);
    else if (cvec)
      rescore_full_kernel<HME_F32, true><<<grid, 256, 0, s>>>(X, d, ldx, C, K, hdr, full_rows, keys_end);
    else
      rescore_full_kernel<HME_F32, false><<<grid, 256, 0, s>>>(X, d, ldx, C, K, hdr, full_rows, keys_end);
  }
  if (!row_path) rescore_full_finish_kernel<<<gfin, 256, 0, s>>>(labels, mind, hdr, full_rows, keys_end);
  count_launch(row_path ? 2 : 3);
  return cudaGetLastError();
}

}  // namespace hme
