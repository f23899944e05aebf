// hme_common.cuh -- internal declarations shared by the CUDA translation units
// of libhme: workspace layout, status bits, launch bookkeeping and the inline
// PTX wrappers (mbarrier, TMA, tcgen05) the sm_103a kernels use.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>
#include <stddef.h>

#include "../../include/hme.h"

namespace hme {

// ---------------------------------------------------------------------------
// status word (first 256 bytes of every workspace)
// ---------------------------------------------------------------------------
enum : uint32_t {
  kStatusBadLabel = 1u << 0,
  kStatusTimeout = 1u << 1,
  kStatusBadTag = 1u << 2,
};

struct Header {          // lives at ws + 0, 256 bytes
  uint32_t status;       // OR of kStatus* bits
  uint32_t rescore_count;  // near-tie rows queued with their two candidates
  uint32_t kpp_choice;   // k-means++: candidate picked in the current round
  uint32_t rescore_full_count;  // near-tie rows queued for a comparison with all K centres
  double objective;      // fp64 objective accumulator of hme_assign
  uint32_t wait_where;   // which bounded wait expired (diagnostic)
  uint32_t cn_max_bits;  // max_k ||c_k||^2 of the prepared centres (float bits; values are >= 0)
  uint32_t moved_rows;   // incremental centre update: rows that changed label (diagnostic)
  uint32_t pad1[55];
};
static_assert(sizeof(Header) == 256, "header is 256 bytes");

constexpr int kBM = 128;        // rows per assign tile (tcgen05 M)
constexpr int kBK = 64;         // bf16 elements per stage k-block (one 128-byte swizzle row)
constexpr int kMaxBN = 256;     // centres per tcgen05 N-chunk
constexpr int kMaxK = 16384;
// small batches: at most kSplitRows rows (the row tiles of one wave) spread
// their N-chunks over at most kMaxSlices CTAs each
constexpr int64_t kSplitRows = 152 * 128;
constexpr int kMaxSlices = 16;
constexpr int kMaxD = 16384;

// ---------------------------------------------------------------------------
// workspace layout
// ---------------------------------------------------------------------------
struct AssignGeom {
  int d, K, dtype;
  int ldp;        // row stride (elements) of the bf16 copies
  int BN;         // centres per N-chunk (multiple of 16, <= 256)
  int nchunks;    // ceil(K / BN)
  int Kp;         // nchunks * BN
  int nprod;      // 1 (bf16 features) or 3 (fp32 features, split products)
  int mt;         // 128-row tiles per CTA sharing each centre stage (1 or 2)
  bool ares;      // A rows resident in shared memory across N-chunks
  bool tf32;      // fp32 features read as tf32 operands (kind::tf32, one product)
  int kblk;       // elements per k-block: 64 (bf16 operands) or 32 (tf32)
  int ldc;        // row stride (elements) of the prepared centres: ldp (bf16) or d rounded to 4 (fp32)
  int nbuf;       // TMEM accumulator buffers (1 or 2)
};

AssignGeom assign_geom(int d, int K, int dtype, bool tf32 = false);

struct PartLayout {
  int64_t tile;     // items per partition tile (one CTA each), a multiple of kPartChunk
  int64_t ntiles;
  int b0, b1, b2;   // digit bits of the chunk sort's passes (0: no such pass)
  size_t tilecnt;   // int32[ntiles * K]
  size_t hist;      // int64[K]
  size_t offs;      // int64[K + 1]
  size_t tagcnt;    // tag lists: int64[ntiles * K] tile tag counts (0: no room for tag lists)
  size_t tag_hist;  // tag lists: int64[K]
  size_t tag_base;  // tag lists: int64[K + 1]
  size_t end;
};
constexpr int kPartChunk = 4096;  // items a partition CTA sorts in shared memory per step
PartLayout part_layout(size_t base, int64_t N, int K, bool tags = false);

struct Layout {
  size_t xn;        // f32[N]
  size_t xhi, xlo;  // bf16[N * ldp] (fp32 features only)
  size_t cb_hi, cb_lo;  // bf16[Kp * ldp]
  size_t cn;        // f32[Kp]
  size_t flagged;   // int32[3N]: near-tie rows queued with their two candidates
  size_t full_rows; // int32[N]: near-tie rows queued for all K centres
  size_t perm, slab;  // int32[N] each: sorted order of the labels (update)
  size_t split;     // float4[min(N, kSplitRows) * kMaxSlices]: row states of centre slices (small batches)
  PartLayout part;  // partition scratch (update / route)
  size_t sums;      // f64[K * d]: per-cluster sums (kept between centre updates)
  size_t counts;    // i64[K]: per-cluster counts (kept between centre updates)
  size_t x2sum;     // f64: sum of ||x||^2 (kept between centre updates)
  size_t delta_k;   // int32[4K] + int64[2]: counts, cursors and totals of the incremental update
  size_t delta_mat; // int32[delta_tiles(N) * 2K]: its per-tile counts
  size_t reseed;    // u64[64 * selecting warps]: re-seed candidate keys
  size_t kpp_rows;  // int32[m]
  size_t kpp_d2;    // f64[m]
  size_t kpp_part;  // f64[blocks]
  size_t total;
};
Layout feature_layout(int64_t N, int d, int K, int dtype, int64_t kpp_m);

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// ---------------------------------------------------------------------------
// host helpers (api.cu)
// ---------------------------------------------------------------------------
int fail(int code, const char *fmt, ...);
int cuda_fail(cudaError_t e, const char *what);
void count_launch(int n = 1);
int num_sms();
uint64_t wait_limit_ns();

// ---------------------------------------------------------------------------
// launchers (one per translation unit)
// ---------------------------------------------------------------------------
cudaError_t launch_prep_features(const void *X, int64_t N, int d, int64_t ldx, int dtype, const AssignGeom &g,
                                 float *xn, __nv_bfloat16 *xhi, __nv_bfloat16 *xlo, cudaStream_t s);
// chi: bf16 rows of bf16(c) or of the split's hi part; for tf32 geometry fp32
// rows of tf32-rounded c (pitch g.ldc).  clo: the split's lo part (fp32
// features, three products) or unused.
cudaError_t launch_prep_centres(const float *C, const AssignGeom &g, void *chi, __nv_bfloat16 *clo, float *cn,
                                Header *hdr, cudaStream_t s);
// part: scratch of small batches (the Layout's split region), or NULL.
int launch_assign(const void *Xa, const void *Xb, int64_t N, int64_t lda, const AssignGeom &g,
                  const void *chi, const __nv_bfloat16 *clo, const float *cn, const float *xn,
                  int32_t *labels, float *mind, Header *hdr, int32_t *flagged, int32_t *full_rows, float4 *part,
                  cudaStream_t s);
// fp32 features with one N-chunk, split to bf16 hi/lo inside the kernel (no
// preparation pass); eligible when X is 16-byte aligned and ldx % 4 == 0.
// Optional outputs: with xhi/xlo/xn set (all or none) the kernel also writes
// the split rows (pitch g.ldp) and their norms, the layout of a preparation
// pass.  With z set it is a projection instead of an assign: it writes
// z[i * ldz + j] = x_i.c_j - cn[j] for j < zcols and touches no label, mind
// or queue.
struct SplitOut {
  __nv_bfloat16 *xhi = nullptr, *xlo = nullptr;
  float *xn = nullptr;
  float *z = nullptr;
  int64_t ldz = 0;
  int zcols = 0;
};
bool split_eligible(const void *X, int64_t ldx, const AssignGeom &g);
int launch_assign_split(const float *X, int64_t N, int64_t ldx, const AssignGeom &g, const __nv_bfloat16 *chi,
                        const __nv_bfloat16 *clo, const float *cn, int32_t *labels, float *mind, Header *hdr,
                        int32_t *flagged, int32_t *full_rows, const SplitOut &out, cudaStream_t s);
// bf16 matrix rows x cols (row stride ld elements), box = box_rows x 64
// columns, 128-byte swizzle (the operand layout of the tcgen05 kernels).
int make_bf16_map(CUtensorMap *m, const void *ptr, uint64_t rows, uint64_t cols, uint64_t ld, uint32_t box_rows);

cudaError_t launch_rescore(const void *X, int64_t N, int d, int64_t ldx, int dtype, const float *C, int K,
                           int32_t *labels, float *mind, Header *hdr, int32_t *flagged,
                           const int32_t *full_rows, cudaStream_t s);
// CSR tag lists that move with their points (hme_partition).
struct TagLists {
  const int64_t *tag_off;  // int64[N + 1]
  const int32_t *tags;
  int64_t *tag_off_out;    // int64[N + 1]
  int32_t *tags_out;
};
// The stable partition (partition.cu).  tl: tag lists moved with their
// points (pl must come from part_layout(..., tags = true)), or NULL.
cudaError_t launch_partition(const int32_t *labels, int64_t N, int K, const PartLayout &pl, char *ws,
                             int64_t *hist, int64_t *offsets, int32_t *perm, int32_t *sorted_labels, Header *hdr,
                             cudaStream_t s, const TagLists *tl = nullptr);
// Per-cluster state carried by the workspace from one centre update to the next.
struct UpdateState {
  double *sums;     // fp64[K * d]: S_k = sum of the rows with label k
  int64_t *counts;  // int64[K]: n_k
  double *x2sum;    // sum_i ||x_i||^2 of the rows with a valid label
};
// Scratch of the incremental update (regions the assign queues and the sort
// order also use; never live at the same time).
struct DeltaScratch {
  int32_t *hist_add, *hist_sub;  // int32[K] each, adjacent (hist_sub = hist_add + K)
  int32_t *cur_add, *cur_sub;    // int32[K] each
  int64_t *totals;               // int64[2]: rows to add, rows to subtract
  int32_t *add_rows, *add_lab, *sub_rows, *sub_lab;  // int32[N] each
  unsigned long long *cand;      // re-seed candidates: 64 keys per selecting warp
  int32_t *mat;                  // int32[delta_tiles(N) * 2K]: changed rows per (tile, bucket)
};
// The calling thread's current CUDA context (NULL if none or unavailable).
void *current_context_handle();
// Row tiles of the incremental update's count and fill (at most 304).
int64_t delta_tiles(int64_t N);
// prev_labels == nullptr: full pass (perm / sorted_labels / hist / valid_total
// from the partition of labels); otherwise an incremental update from the
// state left by a call with prev_labels.
cudaError_t launch_update(const void *X, int64_t N, int d, int64_t ldx, int dtype, const int32_t *labels,
                          const int32_t *prev_labels, const int32_t *perm, const int32_t *sorted_labels,
                          const int64_t *hist, const int64_t *valid_total, const float *mind, int K,
                          UpdateState st, DeltaScratch ds, float *C, int64_t *counts_out, int32_t *n_reseeded,
                          Header *hdr, cudaStream_t s);
cudaError_t launch_update_finish(const void *X, int64_t N, int d, int64_t ldx, int dtype, const float *mind, int K,
                                 UpdateState st, DeltaScratch ds, float *C, int64_t *counts_out, int32_t *n_reseeded,
                                 Header *hdr, cudaStream_t s);
cudaError_t launch_update_add(const void *X, int64_t n, int d, int64_t ldx, int dtype, const int32_t *perm,
                              const int32_t *sorted_labels, const int64_t *hist, const int64_t *valid_total, int K,
                              UpdateState st, bool reset, cudaStream_t s);
cudaError_t launch_kmeanspp(const void *X, int64_t N, int d, int64_t ldx, int dtype, int K, uint64_t seed,
                            int64_t m, bool subsample, float *C_out, int32_t *rows, double *d2, double *part,
                            Header *hdr, cudaStream_t s);
// Tag statistics of a clustering (tags.cu); scratch: chunk_start int64[K + 1],
// colsums double[kTagSlices * 2 V].
constexpr int kTagSlices = 16;
cudaError_t launch_tag_hist(const int64_t *offsets, const int64_t *tag_off, const int32_t *tags, int K, int V,
                            int64_t *chunk_start, double *colsums, int64_t *counts, double *sparsity, Header *hdr,
                            cudaStream_t s);
// PCA (pca.cu): see the file header for the steps.
constexpr int64_t kCovSub = 512;  // rows per fp32 (TMEM) accumulation of the covariance
constexpr int kCovFlush = 16;     // sub-range sums per covariance work unit (fp32 register accumulation)
constexpr int kJacobiMaxSweeps = 40;
struct PcaGeom {
  int64_t N;
  int d, r;
  int n;           // Jacobi order: d rounded up to a multiple of 64
  int64_t ldn;     // rows of the transposed split, padded: nchunks * R
  int mi, ntiles;  // 128-feature tiles along d; upper-triangle tiles
  int64_t R, nchunks, nslabs;  // rows per covariance work unit (= rows per block of the transposed split),
                               // blocks (= units per tile), column-sum slabs
};
PcaGeom pca_geom(int64_t N, int d, int r);
cudaError_t launch_pca_mean(const float *X, const PcaGeom &g, int64_t ldx, double *slab_sums, double *mean64,
                            float *mean32, cudaStream_t s);
// centred transposed split, tcgen05 covariance partials, fp64 reduction into
// cov (d x d, may be null) and A (fp32, order g.n)
int launch_pca_cov(const float *X, const PcaGeom &g, int64_t ldx, const float *mean32, __nv_bfloat16 *yh,
                   __nv_bfloat16 *yl, float *part, double *cov, float *A, Header *hdr, cudaStream_t s);
// Jacobi sweeps on A0 (synchronises s once per sweep), then the r leading
// components (rows of W, r x d) and their variances (may be null)
int run_pca_jacobi(const PcaGeom &g, float *A0, float *V0, float *Qbuf, double *acc, int32_t *order, float *W,
                   float *variances, int *sweeps_out, cudaStream_t s);
constexpr int kPcaMaxFitD = 8192;
cudaError_t launch_pca_zoff(const float *mean, const float *W, int d, int r, int Kp, float *zoff, cudaStream_t s);
cudaError_t launch_debug_wait(uint64_t timeout_ns, Header *hdr, cudaStream_t s);
int64_t kpp_candidates(int64_t N, int K, int method);
constexpr int kMaxSms = 256;  // bound used to size the re-seed candidate region
int64_t kpp_blocks(int64_t m);

// ---------------------------------------------------------------------------
// device-side PTX wrappers
// ---------------------------------------------------------------------------
#ifdef __CUDACC__

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count));
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.release.cta.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cta.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait on an mbarrier phase.  Gives up after limit_ns of global time,
// records kStatusTimeout (and where) in the header and returns false; the
// caller then leaves its loop so that the kernel still ends.
__device__ __forceinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity, uint64_t limit_ns,
                                                  Header *hdr, uint32_t where) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  uint32_t spins = 0;
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((++spins & 63u) == 0 && global_timer_ns() - t0 > limit_ns) {
      atomicOr(&hdr->status, (uint32_t)kStatusTimeout);
      atomicExch(&hdr->wait_where, where);
      return false;
    }
  }
}

// TMA: 2-D tiled bulk load global -> shared, completion counted on an mbarrier.
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *map, uint32_t bar, int32_t c0,
                                            int32_t c1, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(bar), "l"(policy)
      : "memory");
}

// TMA: 3-D tiled bulk load global -> shared (coordinates innermost first).
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap *map, uint32_t bar, int32_t c0,
                                            int32_t c1, int32_t c2, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3, %4}], [%5], %6;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(bar), "l"(policy)
      : "memory");
}

// Shared -> global tiled store (bulk-group completion); the writing threads
// fence their generic-proxy stores with fence_proxy_async_smem() first.
__device__ __forceinline__ void tma_store_2d(const CUtensorMap *map, uint32_t src, int32_t c0, int32_t c1) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(src), "r"(c0), "r"(c1)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// the shared-memory sources of all committed bulk stores have been read
__device__ __forceinline__ void bulk_wait_read_all() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
// all committed bulk stores are complete
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void st_shared_u4(uint32_t saddr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};" ::"r"(saddr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}

__device__ __forceinline__ void prefetch_tensormap(const CUtensorMap *map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

__device__ __forceinline__ uint64_t l2_policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

__device__ __forceinline__ uint64_t l2_policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}

// ---- tcgen05 (5th-generation tensor cores, accumulators in TMEM) ----------

__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
               : "memory");
}

__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}

__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// D[tmem] (+)= A[smem desc] x B[smem desc]^T, kind::f16 (bf16 in, fp32 accumulate).
__device__ __forceinline__ void tc_mma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// D[tmem] (+)= A[smem desc] x B[smem desc]^T, kind::tf32 (fp32 words in shared
// memory read as tf32, fp32 accumulate); K = 8 per instruction, so a 32-byte
// step along k is one instruction, as for kind::f16.
__device__ __forceinline__ void tc_mma_tf32(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// D[tmem] (+)= A[tmem] x B[smem desc]^T, kind::f16, A read from tensor memory:
// row m of A in lane m, 16-bit elements packed in pairs along k into 32-bit
// columns (element 2w in the low half of column w).
__device__ __forceinline__ void tc_mma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                               uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive (once) on an mbarrier when all previously issued tcgen05 ops of this thread complete.
__device__ __forceinline__ void tc_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
               : "memory");
}

// 32 lanes x 32 bits, 16 consecutive columns: thread t of the warp gets lane
// (quarter*32 + t), columns col .. col+15.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}

__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// Wait for outstanding tcgen05.ld and tie the 16 destination registers to the
// wait, so that no use of them can be scheduled before it.
__device__ __forceinline__ void tmem_ld_wait(uint32_t (&r)[16]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]),
                 "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]), "+r"(r[15])
               :
               : "memory");
}

// 32 lanes x 32 bits, 16 consecutive columns from registers: thread t of the
// warp writes lane (quarter*32 + t), columns col .. col+15.
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t *r) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]),
      "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}

__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

__device__ __forceinline__ float4 ld_shared_f4(uint32_t saddr) {
  float4 v;
  asm volatile("ld.shared.v4.f32 {%0,%1,%2,%3}, [%4];" : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "r"(saddr));
  return v;
}

// Shared-memory matrix descriptor for a K-major operand stored in the 128-byte
// swizzled layout that TMA writes with CU_TENSOR_MAP_SWIZZLE_128B: rows of 128
// bytes, 8-row groups 1024 bytes apart (stride byte offset), descriptor
// version 1 (bit 46), layout type 2 = SWIZZLE_128B (bits 61-63).  The leading
// byte offset is unused for this layout.
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t saddr) {
  uint64_t desc = 0;
  desc |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  desc |= (uint64_t)(16u >> 4) << 16;
  desc |= (uint64_t)(1024u >> 4) << 32;
  desc |= (uint64_t)1 << 46;
  desc |= (uint64_t)2 << 61;
  return desc;
}

// Instruction descriptor, kind::f16: D fp32 (bits 4-5 = 1), A bf16 (bits 7-9 = 1),
// B bf16 (bits 10-12 = 1), both K-major (bits 15, 16 = 0), N >> 3 at bits 17-22,
// M >> 4 at bits 24-28.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(uint32_t M, uint32_t N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((N >> 3) << 17) | ((M >> 4) << 24);
}
// kind::tf32: A and B format 2 (tf32), fp32 accumulator, both K-major.
__host__ __device__ constexpr uint32_t idesc_tf32_f32(uint32_t M, uint32_t N) {
  return (1u << 4) | (2u << 7) | (2u << 10) | ((N >> 3) << 17) | ((M >> 4) << 24);
}

#endif  // __CUDACC__

}  // namespace hme
