// api.cu -- the extern "C" entry points of libhme (declared in include/hme.h):
// argument checks, the workspace layout, and the order of kernel launches for
// each operation of the gater (Section 2 of the paper: K-means of the
// features, the hard assignment of Eq. 2, each expert's share of the data).
#include "hme_common.cuh"

#include <atomic>
#include <mutex>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>

namespace hme {

namespace {
thread_local char g_err[512] = {0};
std::atomic<int64_t> g_launches{0};
int g_sms[64] = {0};
}  // namespace

int fail(int code, const char *fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return code;
}

int cuda_fail(cudaError_t e, const char *what) {
  return fail(HME_ECUDA, "%s: %s (%s)", what, cudaGetErrorString(e), cudaGetErrorName(e));
}

void count_launch(int n) { g_launches.fetch_add(n, std::memory_order_relaxed); }

int num_sms() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
  if (g_sms[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
    g_sms[dev] = n;
  }
  return g_sms[dev];
}

uint64_t wait_limit_ns() {
  // Every pipeline wait gives up after this much global time (debug override: HME_WAIT_LIMIT_NS).
  static uint64_t v = [] {
    const char *e = getenv("HME_WAIT_LIMIT_NS");
    if (e && *e) {
      unsigned long long x = strtoull(e, nullptr, 10);
      if (x >= 1000 && x <= 60000000000ull) return (uint64_t)x;
    }
    return (uint64_t)2000000000ull;
  }();
  return v;
}

// Tile shape of the assign kernel.  Every 128-row tile re-reads all centre
// tiles from L2, so for bf16 features (one product, tensor-bound when K is
// large) two row tiles share each centre stage (MT = 2): up to 256 centres per
// N-chunk, single-buffered in TMEM when 2 x BN needs all 512 columns.  With
// several N-chunks and d <= 256 the CTA's 128 rows stay resident in shared
// memory (ARES, MT = 1) and the chunks hold 256 centres, double-buffered: with
// so short a contraction the single MMA-issuing thread, not L2, sets the pace,
// and N = 256 halves the MMAs it issues per flop (MT = 2 with 128-centre
// chunks measured 114 against 96 ms per assign at N = 5e7, d = 256, K = 4096).
// fp32 features (three products, 2 operands per side) keep MT = 1.
AssignGeom assign_geom(int d, int K, int dtype, bool tf32) {
  AssignGeom g;
  g.d = d;
  g.K = K;
  g.dtype = dtype;
  g.ldp = (d + 7) / 8 * 8;
  g.tf32 = tf32 && dtype == HME_F32;
  g.nprod = dtype == HME_F32 && !g.tf32 ? 3 : 1;
  g.kblk = g.tf32 ? 32 : kBK;
  g.ldc = g.tf32 ? (d + 3) / 4 * 4 : g.ldp;
  const int num_kb = (d + g.kblk - 1) / g.kblk;
  int max_bn = kMaxBN;
  g.mt = 1;
  g.ares = false;
  if (g.tf32) {
    // one tf32 product per k-step: two row tiles share each centre stage
    // (half the L2 reads of centres per row), 128-centre chunks so that both
    // accumulators fit TMEM twice (the epilogue overlaps the next MMAs)
    g.mt = 2;
    max_bn = kMaxBN / 2;
  } else if (g.nprod == 1) {
    g.mt = 2;
    if (K > kMaxBN && num_kb * (kBM * kBK * 2) <= 64 * 1024) {
      g.ares = true;
      g.mt = 1;
    }
  }
  g.nchunks = (K + max_bn - 1) / max_bn;
  const int per = (K + g.nchunks - 1) / g.nchunks;
  g.BN = (per + 15) / 16 * 16;
  g.Kp = g.BN * g.nchunks;
  g.nbuf = (g.mt * g.BN <= 256) ? 2 : 1;
  return g;
}

// HME_ASSIGN_TF32: fp32 features with several N-chunks (K > 256) read
// directly as tf32 operands, when TMA can read them (16-byte aligned rows);
// otherwise, and by default, as the bf16 split.
bool use_tf32(const void *X, int64_t ldx, int K, int dtype, int flags) {
  return (flags & HME_ASSIGN_TF32) && dtype == HME_F32 && K > kMaxBN &&
         (reinterpret_cast<uintptr_t>(X) & 15u) == 0 && ldx % 4 == 0;
}
constexpr int kAssignFlags = HME_ASSIGN_PREPARED | HME_ASSIGN_PREPARE_OUT | HME_ASSIGN_TF32;
bool bad_flags(int flags) {
  return (flags & ~kAssignFlags) ||
         (flags & (HME_ASSIGN_PREPARED | HME_ASSIGN_PREPARE_OUT)) == (HME_ASSIGN_PREPARED | HME_ASSIGN_PREPARE_OUT);
}

Layout feature_layout(int64_t N, int d, int K, int dtype, int64_t kpp_m) {
  const AssignGeom g = assign_geom(d, K, dtype);
  // fp32 features with K > 256 may use either operand form (use_tf32): room for both
  const AssignGeom gt = assign_geom(d, K, dtype, dtype == HME_F32 && K > kMaxBN);
  Layout L;
  size_t off = sizeof(Header);
  auto take = [&](size_t bytes) {
    off = align_up(off, 256);
    const size_t at = off;
    off += bytes;
    return at;
  };
  L.xn = take((size_t)N * 4);
  if (dtype == HME_F32) {
    L.xhi = take((size_t)N * g.ldp * 2);
    L.xlo = take((size_t)N * g.ldp * 2);
  } else {
    L.xhi = L.xlo = 0;
  }
  const size_t cb_split = (size_t)g.Kp * g.ldp * 2;
  const size_t cb_tf32 = gt.tf32 ? (size_t)gt.Kp * gt.ldc * 4 : 0;
  L.cb_hi = take(cb_split > cb_tf32 ? cb_split : cb_tf32);
  L.cb_lo = dtype == HME_F32 ? take((size_t)g.Kp * g.ldp * 2) : 0;
  L.cn = take((size_t)(g.Kp > gt.Kp ? g.Kp : gt.Kp) * 4);
  L.flagged = take((size_t)(N > 0 ? N : 1) * 12);  // (row, best, runner-up) per queued row
  L.full_rows = take((size_t)(N > 0 ? N : 1) * 4);
  L.perm = take((size_t)(N > 0 ? N : 1) * 4);
  L.slab = take((size_t)(N > 0 ? N : 1) * 4);
  L.split = take((size_t)(N < kSplitRows ? (N > 0 ? N : 1) : kSplitRows) * kMaxSlices * 16);
  L.part = part_layout(align_up(off, 256), N, K);
  off = L.part.end;
  L.sums = take((size_t)K * d * 8);
  L.counts = take((size_t)K * 8);
  L.x2sum = take(8);
  L.delta_k = take((size_t)4 * K * 4 + 16);
  L.delta_mat = take((size_t)delta_tiles(N) * 2 * K * 4);
  L.reseed = take((size_t)kMaxSms * 2 * 8 * 64 * 8);  // (2 blocks x 8 warps per SM) x 64 keys
  if (kpp_m > 0) {
    L.kpp_rows = take((size_t)kpp_m * 4);
    L.kpp_d2 = take((size_t)kpp_m * 8);
    L.kpp_part = take((size_t)kpp_blocks(kpp_m) * 8);
  } else {
    L.kpp_rows = L.kpp_d2 = L.kpp_part = 0;
  }
  L.total = align_up(off, 256);
  return L;
}

namespace {

size_t init_bytes(int64_t N, int K) {
  size_t off = sizeof(Header);
  const int64_t m = N;  // upper bound over both methods
  off = align_up(off, 256) + (size_t)m * 4;
  off = align_up(off, 256) + (size_t)m * 8;
  off = align_up(off, 256) + (size_t)kpp_blocks(m) * 8;
  (void)K;
  return align_up(off, 256);
}

int check_common(int64_t N, int d, int K, int dtype) {
  if (N < 0 || N > (int64_t)0x7FFFFFFF) return fail(HME_EINVAL, "N = %lld out of range [0, 2^31)", (long long)N);
  if (d < 1 || d > kMaxD) return fail(HME_EINVAL, "d = %d out of range [1, %d]", d, kMaxD);
  if (K < 1 || K > kMaxK) return fail(HME_EINVAL, "K = %d out of range [1, %d]", K, kMaxK);
  if (dtype != HME_F32 && dtype != HME_BF16) return fail(HME_EINVAL, "dtype = %d is not HME_F32 or HME_BF16", dtype);
  return HME_OK;
}

int check_features(const void *X, int64_t N, int d, int64_t ldx, int dtype, bool tma) {
  if (N > 0 && !X) return fail(HME_EINVAL, "feature pointer is NULL");
  if (ldx < d) return fail(HME_EINVAL, "ldx = %lld < d = %d", (long long)ldx, d);
  if (tma && dtype == HME_BF16) {
    if ((reinterpret_cast<uintptr_t>(X) & 15u) != 0)
      return fail(HME_EINVAL, "bf16 features must start on a 16-byte boundary (TMA)");
    if ((ldx * 2) % 16 != 0)
      return fail(HME_EINVAL, "bf16 row stride ldx = %lld is not a multiple of 8 elements (TMA)", (long long)ldx);
  }
  return HME_OK;
}

int check_ws(void *ws, size_t ws_bytes, size_t need) {
  if (!ws) return fail(HME_EINVAL, "workspace is NULL");
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return fail(HME_EINVAL, "workspace is not 256-byte aligned");
  if (ws_bytes < need)
    return fail(HME_ENOMEM, "workspace of %zu bytes is smaller than the %zu bytes needed", ws_bytes, need);
  return HME_OK;
}

#define HME_TRY(expr)                   \
  do {                                  \
    int _rc = (expr);                   \
    if (_rc != HME_OK) return _rc;      \
  } while (0)

#define HME_CUDA(expr, what)                         \
  do {                                               \
    cudaError_t _e = (expr);                         \
    if (_e != cudaSuccess) return cuda_fail(_e, what); \
  } while (0)

template <typename T>
T *at(void *ws, size_t off) {
  return reinterpret_cast<T *>(static_cast<char *>(ws) + off);
}

int do_prepare(const void *X, int64_t N, int d, int64_t ldx, int dtype, int K, const Layout &L, void *ws,
               cudaStream_t s, int flags = 0) {
  const AssignGeom g = assign_geom(d, K, dtype, use_tf32(X, ldx, K, dtype, flags));
  HME_CUDA(launch_prep_features(X, N, d, ldx, dtype, g, at<float>(ws, L.xn), at<__nv_bfloat16>(ws, L.xhi),
                                at<__nv_bfloat16>(ws, L.xlo), s),
           "prepare features");
  return HME_OK;
}

int launch_assign_prepared(const void *X, int64_t N, int64_t ldx, int dtype, const AssignGeom &g, const Layout &L,
                           void *ws, int32_t *labels, float *mind, Header *hdr, cudaStream_t s);

// prepared: ws holds this X's preparation (hme_prepare_features).  An
// unprepared call on fp32 features that TMA can read splits the rows inside
// the assign kernel (one pass over X); any other unprepared call prepares
// first.  Prepared calls use the prepared operands, which stream at the
// full HBM rate.  prepare_out: an in-kernel split also writes the prepared
// operands to ws (every other unprepared call leaves them there anyway).
int do_assign(const void *X, int64_t N, int d, int64_t ldx, int dtype, const float *C, int K, int32_t *labels,
              float *mind, const Layout &L, void *ws, int flags, cudaStream_t s) {
  const bool prepared = (flags & HME_ASSIGN_PREPARED) != 0, prepare_out = (flags & HME_ASSIGN_PREPARE_OUT) != 0;
  const AssignGeom g = assign_geom(d, K, dtype, use_tf32(X, ldx, K, dtype, flags));
  const bool split = !prepared && split_eligible(X, ldx, g);
  if (!prepared && !split) HME_TRY(do_prepare(X, N, d, ldx, dtype, K, L, ws, s, flags));
  Header *hdr = at<Header>(ws, 0);
  HME_CUDA(launch_prep_centres(C, g, at<void>(ws, L.cb_hi), at<__nv_bfloat16>(ws, L.cb_lo), at<float>(ws, L.cn),
                               hdr, s),
           "prepare centres");
  if (split) {
    SplitOut out;
    if (prepare_out) {
      out.xhi = at<__nv_bfloat16>(ws, L.xhi);
      out.xlo = at<__nv_bfloat16>(ws, L.xlo);
      out.xn = at<float>(ws, L.xn);
    }
    HME_TRY(launch_assign_split(static_cast<const float *>(X), N, ldx, g, at<__nv_bfloat16>(ws, L.cb_hi),
                                at<__nv_bfloat16>(ws, L.cb_lo), at<float>(ws, L.cn), labels, mind, hdr,
                                at<int32_t>(ws, L.flagged), at<int32_t>(ws, L.full_rows), out, s));
  } else {
    HME_TRY(launch_assign_prepared(X, N, ldx, dtype, g, L, ws, labels, mind, hdr, s));
  }
  HME_CUDA(launch_rescore(X, N, d, ldx, dtype, C, K, labels, mind, hdr, at<int32_t>(ws, L.flagged),
                          at<int32_t>(ws, L.full_rows), s),
           "re-score");
  return HME_OK;
}

int launch_assign_prepared(const void *X, int64_t N, int64_t ldx, int dtype, const AssignGeom &g, const Layout &L,
                           void *ws, int32_t *labels, float *mind, Header *hdr, cudaStream_t s) {
  const bool split = g.nprod == 3;  // the prepared bf16 split; else X itself (bf16, or fp32 read as tf32)
  const void *Xa = split ? (const void *)at<__nv_bfloat16>(ws, L.xhi) : X;
  const void *Xb = split ? (const void *)at<__nv_bfloat16>(ws, L.xlo) : X;
  const int64_t lda = split ? g.ldp : ldx;
  HME_TRY(launch_assign(Xa, Xb, N, lda, g, at<void>(ws, L.cb_hi), at<__nv_bfloat16>(ws, L.cb_lo),
                        at<float>(ws, L.cn), at<float>(ws, L.xn), labels, mind, hdr, at<int32_t>(ws, L.flagged),
                        at<int32_t>(ws, L.full_rows), at<float4>(ws, L.split), s));
  return HME_OK;
}

// hme_tag_cluster_hist: header, chunk table int64[K + 1], per-slice column sums double[kTagSlices][2 V]
size_t tag_ws_bytes(int K, int V) {
  return align_up(align_up(sizeof(Header) + (size_t)(K + 1) * sizeof(int64_t), 256) +
                      (size_t)kTagSlices * 2 * V * sizeof(double),
                  256);
}

// hme_kmeans_stream: a chunk's assign/update workspace, then two device chunk
// buffers of dense rows (pitch stream_ld(d) elements: 16-byte rows for TMA).
int64_t stream_ld(int d, int dtype) { return dtype == HME_F32 ? (d + 3) / 4 * 4 : (d + 7) / 8 * 8; }
size_t stream_buf_bytes(int64_t chunk, int d, int dtype) {
  return align_up((size_t)chunk * stream_ld(d, dtype) * (dtype == HME_F32 ? 4 : 2), 256);
}
size_t stream_ws_bytes(int64_t chunk, int d, int K, int dtype) {
  return align_up(feature_layout(chunk, d, K, dtype, 0).total, 256) + 2 * stream_buf_bytes(chunk, d, dtype);
}

int clear_header(void *ws, cudaStream_t s) {
  HME_CUDA(cudaMemsetAsync(ws, 0, sizeof(Header), s), "clear workspace header");
  return HME_OK;
}

// PCA fit (hme_pca_covariance / hme_pca_fit): slab sums, mean, transposed
// split, covariance partial tiles, the Jacobi matrices and small scratch.
struct PcaLayout {
  size_t slab, mean64, mean32, yh, yl, part, A0, V0, qbuf, acc, order, total;
};
PcaLayout pca_layout(int64_t N, int d, int r) {
  const PcaGeom g = pca_geom(N, d, r);
  PcaLayout L;
  size_t off = sizeof(Header);
  auto take = [&](size_t bytes) {
    off = align_up(off, 256);
    const size_t at = off;
    off += bytes;
    return at;
  };
  L.slab = take((size_t)g.nslabs * d * 8);
  L.mean64 = take((size_t)d * 8);
  L.mean32 = take((size_t)d * 4);
  L.yh = take((size_t)d * g.ldn * 2);
  L.yl = take((size_t)d * g.ldn * 2);
  L.part = take((size_t)g.nchunks * g.ntiles * kBM * kBM * 4);
  const size_t nn = (size_t)g.n * g.n * 4;
  L.A0 = take(nn);
  L.V0 = take(nn);
  L.qbuf = take((size_t)(g.n / 64) * 64 * 64 * 4);
  L.acc = take(16);
  L.order = take((size_t)r * 4);
  L.total = align_up(off, 256);
  return L;
}
// hme_pca_transform: the components split to bf16 (hi, lo), their norms and
// the per-component offsets mu.w_j
struct PcaTLayout {
  size_t chi, clo, cn, zoff, total;
};
PcaTLayout pca_t_layout(int d, int r) {
  const AssignGeom g = assign_geom(d, r, HME_F32);
  PcaTLayout L;
  size_t off = sizeof(Header);
  auto take = [&](size_t bytes) {
    off = align_up(off, 256);
    const size_t at = off;
    off += bytes;
    return at;
  };
  L.chi = take((size_t)g.Kp * g.ldp * 2);
  L.clo = take((size_t)g.Kp * g.ldp * 2);
  L.cn = take((size_t)g.Kp * 4);
  L.zoff = take((size_t)g.Kp * 4);
  L.total = align_up(off, 256);
  return L;
}
int check_pca_sizes(int64_t N, int d, int dtype, int r, int64_t min_n) {
  if (dtype != HME_F32) return fail(HME_EINVAL, "PCA takes fp32 features (dtype HME_F32)");
  if (N < min_n || N > (int64_t)0x7FFFFFFF)
    return fail(HME_EINVAL, "N = %lld out of range [%lld, 2^31)", (long long)N, (long long)min_n);
  if (d < 1 || d > kMaxD) return fail(HME_EINVAL, "d = %d out of range [1, %d]", d, kMaxD);
  if (r < 1 || r > d) return fail(HME_EINVAL, "r = %d out of range [1, d = %d]", r, d);
  return HME_OK;
}
int check_pca(const void *X, int64_t N, int d, int64_t ldx, int dtype, int r, int64_t min_n) {
  HME_TRY(check_pca_sizes(N, d, dtype, r, min_n));
  if (N > 0 && !X) return fail(HME_EINVAL, "feature pointer is NULL");
  if (ldx < d) return fail(HME_EINVAL, "ldx = %lld < d = %d", (long long)ldx, d);
  return HME_OK;
}

}  // namespace
// Small routed batches are launch-bound (a dozen kernels of a few
// microseconds each).  A route of at most kGraphRows rows whose arguments --
// every pointer, size, flag and the stream -- repeat those of an earlier call
// is captured once as a CUDA graph (on a stream of the library's own, so that
// any stream of the caller's, the legacy default one included, can replay it)
// and from then on replayed with one launch.  The captured launches depend on
// the arguments only, never on the data, which the kernels read when they
// run.  The first call with a given set of arguments runs directly (a batch
// routed once pays no capture); a capture that fails leaves that set direct.
// The CUDA context is part of the key (a graph cannot outlive its context).
constexpr int64_t kGraphRows = 16384;
constexpr int kGraphSlots = 8;
struct RouteKey {
  const void *Q;
  int64_t B;
  int32_t d;
  int64_t ldq;
  int32_t dtype;
  const float *C;
  int32_t K;
  int32_t flags;
  int32_t *expert;
  int64_t *offsets;
  int32_t *order;
  void *ws;
  size_t ws_bytes;
  void *stream;
  int device = 0;
  void *context = nullptr;  // a graph belongs to the context it was captured in
  bool operator==(const RouteKey &o) const {
    return Q == o.Q && B == o.B && d == o.d && ldq == o.ldq && dtype == o.dtype && C == o.C && K == o.K &&
           flags == o.flags && expert == o.expert && offsets == o.offsets && order == o.order && ws == o.ws &&
           ws_bytes == o.ws_bytes && stream == o.stream && device == o.device && context == o.context;
  }
};
struct RouteGraph {
  RouteKey key{};
  bool used = false;
  bool direct = false;  // capture failed: stay direct
  cudaGraphExec_t exec = nullptr;
  int64_t launches = 0;
  uint64_t stamp = 0;
};
std::mutex g_rg_mu;
RouteGraph g_rg[kGraphSlots];
uint64_t g_rg_clock = 0;
cudaStream_t g_cap_stream[64] = {};

template <typename Body>
int graph_route(RouteKey key, Body &&body, cudaStream_t s) {
  static const bool off = [] {
    const char *e = getenv("HME_NO_GRAPHS");
    return e && *e && *e != '0';
  }();
  if (off || cudaGetDevice(&key.device) != cudaSuccess || key.device < 0 || key.device >= 64) return body(s);
  key.context = current_context_handle();
  if (!key.context) return body(s);
  std::unique_lock<std::mutex> lk(g_rg_mu);
  RouteGraph *slot = nullptr;
  for (auto &g : g_rg)
    if (g.used && g.key == key) slot = &g;
  if (slot && slot->exec) {
    slot->stamp = ++g_rg_clock;
    const cudaGraphExec_t exec = slot->exec;
    const int64_t n = slot->launches;
    lk.unlock();
    HME_CUDA(cudaGraphLaunch(exec, s), "route: graph launch");
    count_launch((int)n);
    return HME_OK;
  }
  if (!slot) {  // first sighting: remember the arguments, run directly
    RouteGraph *victim = &g_rg[0];
    for (auto &g : g_rg)
      if (!g.used || g.stamp < victim->stamp) victim = &g;
    if (victim->exec) cudaGraphExecDestroy(victim->exec);
    *victim = RouteGraph{};
    victim->key = key;
    victim->used = true;
    victim->stamp = ++g_rg_clock;
    lk.unlock();
    return body(s);
  }
  if (slot->direct) {
    lk.unlock();
    return body(s);
  }
  // second sighting: capture on the library's stream, then replay on s
  cudaStream_t &cs = g_cap_stream[key.device];
  if (!cs && cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking) != cudaSuccess) {
    cs = nullptr;
    slot->direct = true;
    lk.unlock();
    return body(s);
  }
  const int64_t before = g_launches.load();
  cudaGraph_t graph = nullptr;
  int rc = HME_OK;
  if (cudaStreamBeginCapture(cs, cudaStreamCaptureModeThreadLocal) == cudaSuccess) {
    rc = body(cs);
    const cudaError_t e = cudaStreamEndCapture(cs, &graph);
    if (e != cudaSuccess && graph) {
      cudaGraphDestroy(graph);
      graph = nullptr;
    }
  }
  cudaGraphExec_t exec = nullptr;
  if (rc == HME_OK && graph && cudaGraphInstantiate(&exec, graph, 0) != cudaSuccess) exec = nullptr;
  if (graph) cudaGraphDestroy(graph);
  cudaGetLastError();  // a failed capture leaves no sticky error behind
  if (!exec) {
    slot->direct = true;
    g_launches.fetch_sub(g_launches.load() - before);  // nothing captured ran
    lk.unlock();
    return rc == HME_OK ? body(s) : rc;
  }
  slot->exec = exec;
  slot->launches = g_launches.load() - before;
  slot->stamp = ++g_rg_clock;
  lk.unlock();
  HME_CUDA(cudaGraphLaunch(exec, s), "route: graph launch");
  return HME_OK;
}

}  // namespace hme

using namespace hme;

extern "C" {

size_t hme_workspace_bytes(int32_t op, int64_t N, int32_t d, int32_t K, int32_t dtype) {
  if (op == HME_OP_PARTITION) {
    if (N < 0 || N > (int64_t)0x7FFFFFFF || K < 1 || K > kMaxK) return 0;
    return align_up(part_layout(sizeof(Header), N, K, true).end, 256);  // room for tag lists
  }
  if (op == HME_OP_STREAM) {  // N is the chunk length
    if (check_common(N, d, K, dtype) != HME_OK || N < 1) return 0;
    return stream_ws_bytes(N, d, K, dtype);
  }
  if (op == HME_OP_PCA) {  // K is the number of components r; N = 0: hme_pca_transform only
    if (check_pca_sizes(N, d, dtype, K, 0) != HME_OK) return 0;
    const size_t t = pca_t_layout(d, K > kMaxBN ? kMaxBN : K).total;
    if (N == 0) return t;
    const size_t f = pca_layout(N, d, K).total;
    return f > t ? f : t;
  }
  if (op == HME_OP_TAG_HIST) {  // d is the vocabulary size V
    if (N < 0 || K < 1 || K > kMaxK || d < 1) return 0;
    return tag_ws_bytes(K, d);
  }
  if (check_common(N, d, K, dtype) != HME_OK) return 0;
  switch (op) {
    case HME_OP_INIT:
      return init_bytes(N, K);
    case HME_OP_ASSIGN:
    case HME_OP_ROUTE:
      return feature_layout(N, d, K, dtype, 0).total;
    default:
      fail(HME_EINVAL, "unknown op %d", op);
      return 0;
  }
}

const char *hme_last_error(void) { return g_err; }

int64_t hme_launch_count(void) { return g_launches.load(); }

int hme_sync_status(void *ws, void *stream) {
  if (!ws) return fail(HME_EINVAL, "workspace is NULL");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  HME_CUDA(cudaStreamSynchronize(s), "synchronize");
  Header h;
  HME_CUDA(cudaMemcpy(&h, ws, sizeof(Header), cudaMemcpyDeviceToHost), "read status");
  if (h.status & kStatusTimeout)
    return fail(HME_ETIMEOUT, "a bounded device wait expired (site %u)", h.wait_where);
  if (h.status & kStatusBadLabel) return fail(HME_EINVAL, "a label outside [0, K) was skipped");
  if (h.status & kStatusBadTag)
    return fail(HME_EINVAL, "a tag outside [0, V) was skipped, or a cluster's tag range was inverted");
  return HME_OK;
}

int hme_kmeans_init(const void *X, int64_t N, int32_t d, int64_t ldx, int32_t dtype, int32_t K, uint64_t seed,
                    int32_t method, float *C_out, void *ws, size_t ws_bytes, void *stream) {
  HME_TRY(check_common(N, d, K, dtype));
  if (N < 1) return fail(HME_EINVAL, "k-means++ needs N >= 1");
  if (method != HME_INIT_KMEANSPP && method != HME_INIT_KMEANSPP_SUBSAMPLE)
    return fail(HME_EINVAL, "unknown init method %d", method);
  HME_TRY(check_features(X, N, d, ldx, dtype, false));
  if (!C_out) return fail(HME_EINVAL, "C_out is NULL");
  HME_TRY(check_ws(ws, ws_bytes, init_bytes(N, K)));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int64_t m = kpp_candidates(N, K, method);
  size_t off = align_up(sizeof(Header), 256);
  int32_t *rows = at<int32_t>(ws, off);
  off = align_up(off + (size_t)m * 4, 256);
  double *d2 = at<double>(ws, off);
  off = align_up(off + (size_t)m * 8, 256);
  double *part = at<double>(ws, off);
  HME_TRY(clear_header(ws, s));
  HME_CUDA(launch_kmeanspp(X, N, d, ldx, dtype, K, seed, m, method == HME_INIT_KMEANSPP_SUBSAMPLE, C_out, rows, d2,
                           part, at<Header>(ws, 0), s),
           "k-means++");
  return HME_OK;
}

int hme_prepare_features(const void *X, int64_t N, int32_t d, int64_t ldx, int32_t dtype, int32_t K, void *ws,
                         size_t ws_bytes, void *stream) {
  HME_TRY(check_common(N, d, K, dtype));
  HME_TRY(check_features(X, N, d, ldx, dtype, true));
  const Layout L = feature_layout(N, d, K, dtype, 0);
  HME_TRY(check_ws(ws, ws_bytes, L.total));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  HME_TRY(clear_header(ws, s));
  return do_prepare(X, N, d, ldx, dtype, K, L, ws, s);
}

int hme_assign(const void *X, int64_t N, int32_t d, int64_t ldx, int32_t dtype, const float *C, int32_t K,
               int32_t flags, int32_t *labels_out, float *mind_out, double *objective_out, void *ws,
               size_t ws_bytes, void *stream) {
  HME_TRY(check_common(N, d, K, dtype));
  HME_TRY(check_features(X, N, d, ldx, dtype, true));
  if (!C) return fail(HME_EINVAL, "C is NULL");
  if (N > 0 && !labels_out) return fail(HME_EINVAL, "labels_out is NULL");
  if (bad_flags(flags)) return fail(HME_EINVAL, "unknown flags 0x%x", flags);
  const Layout L = feature_layout(N, d, K, dtype, 0);
  HME_TRY(check_ws(ws, ws_bytes, L.total));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  HME_TRY(clear_header(ws, s));
  HME_TRY(do_assign(X, N, d, ldx, dtype, C, K, labels_out, mind_out, L, ws, flags, s));
  if (objective_out)
    HME_CUDA(cudaMemcpyAsync(objective_out, &at<Header>(ws, 0)->objective, sizeof(double), cudaMemcpyDeviceToDevice,
                             s),
             "copy objective");
  return HME_OK;
}

int hme_assign_rows(const void *X, int64_t N, int64_t row0, int64_t row1, int32_t d, int64_t ldx, int32_t dtype,
                    const float *C, int32_t K, int32_t flags, int32_t *labels_out, float *mind_out,
                    double *objective_out, void *ws, size_t ws_bytes, void *stream) {
  HME_TRY(check_common(N, d, K, dtype));
  if (row0 < 0 || row1 < row0 || row1 > N)
    return fail(HME_EINVAL, "rows [%lld, %lld) are not inside [0, N = %lld)", (long long)row0, (long long)row1,
                (long long)N);
  if (bad_flags(flags)) return fail(HME_EINVAL, "unknown flags 0x%x", flags);
  if (!C) return fail(HME_EINVAL, "C is NULL");
  if (row1 > row0 && !labels_out) return fail(HME_EINVAL, "labels_out is NULL");
  const int64_t esz = dtype == HME_F32 ? 4 : 2;
  const void *Xr = X ? static_cast<const char *>(X) + row0 * ldx * esz : nullptr;
  HME_TRY(check_features(Xr, row1 - row0, d, ldx, dtype, true));
  const Layout L = feature_layout(N, d, K, dtype, 0);
  HME_TRY(check_ws(ws, ws_bytes, L.total));
  // the preparation of rows [row0, row1) sits at their place in the N-row layout
  const AssignGeom g = assign_geom(d, K, dtype);
  Layout Lr = L;
  Lr.xn += (size_t)row0 * 4;
  if (dtype == HME_F32) {
    Lr.xhi += (size_t)row0 * g.ldp * 2;
    Lr.xlo += (size_t)row0 * g.ldp * 2;
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  HME_TRY(clear_header(ws, s));
  HME_TRY(do_assign(Xr, row1 - row0, d, ldx, dtype, C, K, labels_out ? labels_out + row0 : nullptr,
                    mind_out ? mind_out + row0 : nullptr, Lr, ws, flags, s));
  if (objective_out)
    HME_CUDA(cudaMemcpyAsync(objective_out, &at<Header>(ws, 0)->objective, sizeof(double), cudaMemcpyDeviceToDevice,
                             s),
             "copy objective");
  return HME_OK;
}

int hme_update_centroids(const void *X, int64_t N, int32_t d, int64_t ldx, int32_t dtype, const int32_t *labels,
                         const int32_t *prev_labels, const float *mind, int32_t K, float *C_inout,
                         int64_t *counts_out, int32_t *n_reseeded_out, double *objective_out, void *ws,
                         size_t ws_bytes, void *stream) {
  HME_TRY(check_common(N, d, K, dtype));
  HME_TRY(check_features(X, N, d, ldx, dtype, false));
  if (!C_inout) return fail(HME_EINVAL, "C_inout is NULL");
  if (N > 0 && !labels) return fail(HME_EINVAL, "labels is NULL");
  const Layout L = feature_layout(N, d, K, dtype, 0);
  HME_TRY(check_ws(ws, ws_bytes, L.total));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  HME_TRY(clear_header(ws, s));
  Header *hdr = at<Header>(ws, 0);
  int64_t *hist = at<int64_t>(ws, L.part.hist);
  int64_t *offs = at<int64_t>(ws, L.part.offs);
  int32_t *perm = at<int32_t>(ws, L.perm);
  int32_t *slab = at<int32_t>(ws, L.slab);
  if (!prev_labels)
    HME_CUDA(launch_partition(labels, N, K, L.part, static_cast<char *>(ws), hist, offs, perm, slab, hdr, s),
             "update: sort labels");
  UpdateState st{at<double>(ws, L.sums), at<int64_t>(ws, L.counts), at<double>(ws, L.x2sum)};
  int32_t *dk = at<int32_t>(ws, L.delta_k);
  int32_t *fl = at<int32_t>(ws, L.flagged);  // int32[3N]; free while no assign is in flight on this ws
  DeltaScratch ds{dk, dk + K, dk + 2 * K, dk + 3 * K, reinterpret_cast<int64_t *>(dk + 4 * K),
                  perm, slab, fl, fl + N, at<unsigned long long>(ws, L.reseed), at<int32_t>(ws, L.delta_mat)};
  HME_CUDA(launch_update(X, N, d, ldx, dtype, labels, prev_labels, perm, slab, hist, offs + K, mind, K, st, ds,
                         C_inout, counts_out, n_reseeded_out, hdr, s),
           "update: centres");
  if (objective_out)
    HME_CUDA(cudaMemcpyAsync(objective_out, &hdr->objective, sizeof(double), cudaMemcpyDeviceToDevice, s),
             "copy objective");
  return HME_OK;
}

int hme_partition(const int32_t *labels, int64_t N, int32_t K, int64_t *hist_out, int64_t *offsets_out,
                  int32_t *perm_out, int32_t *sorted_labels_out, const int64_t *tag_off, const int32_t *tags,
                  int64_t *tag_off_out, int32_t *tags_out, void *ws, size_t ws_bytes, void *stream) {
  if (N < 0 || N > (int64_t)0x7FFFFFFF) return fail(HME_EINVAL, "N = %lld out of range", (long long)N);
  if (K < 1 || K > kMaxK) return fail(HME_EINVAL, "K = %d out of range [1, %d]", K, kMaxK);
  if (!hist_out || !offsets_out) return fail(HME_EINVAL, "hist_out / offsets_out is NULL");
  if (N > 0 && (!labels || !perm_out)) return fail(HME_EINVAL, "labels / perm_out is NULL");
  const int ntag = (tag_off != nullptr) + (tags != nullptr) + (tag_off_out != nullptr) + (tags_out != nullptr);
  if (ntag != 0 && ntag != 4) return fail(HME_EINVAL, "tag arrays must be all NULL or all set");
  const PartLayout pl = part_layout(sizeof(Header), N, K, ntag == 4);
  HME_TRY(check_ws(ws, ws_bytes, align_up(pl.end, 256)));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  HME_TRY(clear_header(ws, s));
  const TagLists tl{tag_off, tags, tag_off_out, tags_out};
  HME_CUDA(launch_partition(labels, N, K, pl, static_cast<char *>(ws), hist_out, offsets_out, perm_out,
                            sorted_labels_out, at<Header>(ws, 0), s, ntag == 4 ? &tl : nullptr),
           "partition");
  return HME_OK;
}

int hme_route(const void *Q, int64_t B, int32_t d, int64_t ldq, int32_t dtype, const float *C, int32_t K,
              int32_t flags, int32_t *expert_out, int64_t *offsets_out, int32_t *order_out, void *ws, size_t ws_bytes,
              void *stream) {
  HME_TRY(check_common(B, d, K, dtype));
  HME_TRY(check_features(Q, B, d, ldq, dtype, true));
  if (!C) return fail(HME_EINVAL, "C is NULL");
  if (!offsets_out) return fail(HME_EINVAL, "offsets_out is NULL");
  if (B > 0 && (!expert_out || !order_out)) return fail(HME_EINVAL, "expert_out / order_out is NULL");
  if (bad_flags(flags)) return fail(HME_EINVAL, "unknown flags 0x%x", flags);
  const Layout L = feature_layout(B, d, K, dtype, 0);
  HME_TRY(check_ws(ws, ws_bytes, L.total));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  auto body = [&](cudaStream_t cs) -> int {
    HME_TRY(clear_header(ws, cs));
    HME_TRY(do_assign(Q, B, d, ldq, dtype, C, K, expert_out, nullptr, L, ws, flags, cs));
    HME_CUDA(launch_partition(expert_out, B, K, L.part, static_cast<char *>(ws), at<int64_t>(ws, L.part.hist),
                              offsets_out, order_out, nullptr, at<Header>(ws, 0), cs),
             "route: partition");
    return HME_OK;
  };
  if (B > 0 && B <= kGraphRows) {
    const RouteKey key{Q, B, d, ldq, dtype, C, K, flags, expert_out, offsets_out, order_out, ws, ws_bytes, stream};
    return graph_route(key, body, s);
  }
  return body(s);
}

int hme_tag_cluster_hist(const int64_t *offsets, const int64_t *tag_off, const int32_t *tags, int64_t N, int32_t K,
                         int32_t V, int64_t *counts_out, double *sparsity_out, void *ws, size_t ws_bytes,
                         void *stream) {
  if (N < 0 || N > (int64_t)0x7FFFFFFF) return fail(HME_EINVAL, "N = %lld out of range", (long long)N);
  if (K < 1 || K > kMaxK) return fail(HME_EINVAL, "K = %d out of range [1, %d]", K, kMaxK);
  if (V < 1) return fail(HME_EINVAL, "V = %d must be positive", V);
  if (!offsets || !tag_off || !counts_out) return fail(HME_EINVAL, "offsets / tag_off / counts_out is NULL");
  if (!tags && N > 0) return fail(HME_EINVAL, "tags is NULL");
  HME_TRY(check_ws(ws, ws_bytes, tag_ws_bytes(K, V)));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  HME_TRY(clear_header(ws, s));
  const size_t sums_at = align_up(sizeof(Header) + (size_t)(K + 1) * sizeof(int64_t), 256);
  HME_CUDA(launch_tag_hist(offsets, tag_off, tags, K, V, at<int64_t>(ws, sizeof(Header)), at<double>(ws, sums_at),
                           counts_out, sparsity_out, at<Header>(ws, 0), s),
           "tag statistics");
  return HME_OK;
}

int hme_pca_covariance(const void *X, int64_t N, int32_t d, int64_t ldx, int32_t dtype, double *mean_out,
                       double *cov_out, void *ws, size_t ws_bytes, void *stream) {
  HME_TRY(check_pca(X, N, d, ldx, dtype, 1, 1));
  if (!mean_out || !cov_out) return fail(HME_EINVAL, "mean_out / cov_out is NULL");
  const PcaLayout L = pca_layout(N, d, 1);
  HME_TRY(check_ws(ws, ws_bytes, L.total));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  HME_TRY(clear_header(ws, s));
  const PcaGeom g = pca_geom(N, d, 1);
  const float *Xf = static_cast<const float *>(X);
  HME_CUDA(launch_pca_mean(Xf, g, ldx, at<double>(ws, L.slab), at<double>(ws, L.mean64), at<float>(ws, L.mean32), s),
           "pca: mean");
  HME_TRY(launch_pca_cov(Xf, g, ldx, at<float>(ws, L.mean32), at<__nv_bfloat16>(ws, L.yh),
                         at<__nv_bfloat16>(ws, L.yl), at<float>(ws, L.part), cov_out, at<float>(ws, L.A0),
                         at<Header>(ws, 0), s));
  HME_CUDA(cudaMemcpyAsync(mean_out, at<double>(ws, L.mean64), (size_t)d * 8, cudaMemcpyDeviceToDevice, s),
           "pca: copy mean");
  return HME_OK;
}

int hme_pca_fit(const void *X, int64_t N, int32_t d, int64_t ldx, int32_t dtype, int32_t r, float *mean_out,
                float *components_out, float *variances_out, int32_t *sweeps_out, void *ws, size_t ws_bytes,
                void *stream) {
  HME_TRY(check_pca(X, N, d, ldx, dtype, r, 1));
  if (d > kPcaMaxFitD) return fail(HME_EINVAL, "d = %d: hme_pca_fit takes d <= %d", d, kPcaMaxFitD);
  if (!mean_out || !components_out) return fail(HME_EINVAL, "mean_out / components_out is NULL");
  const PcaLayout L = pca_layout(N, d, r);
  HME_TRY(check_ws(ws, ws_bytes, L.total));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  HME_TRY(clear_header(ws, s));
  const PcaGeom g = pca_geom(N, d, r);
  const float *Xf = static_cast<const float *>(X);
  HME_CUDA(launch_pca_mean(Xf, g, ldx, at<double>(ws, L.slab), at<double>(ws, L.mean64), at<float>(ws, L.mean32), s),
           "pca: mean");
  HME_TRY(launch_pca_cov(Xf, g, ldx, at<float>(ws, L.mean32), at<__nv_bfloat16>(ws, L.yh),
                         at<__nv_bfloat16>(ws, L.yl), at<float>(ws, L.part), nullptr, at<float>(ws, L.A0),
                         at<Header>(ws, 0), s));
  int sweeps = 0;
  const int rc = run_pca_jacobi(g, at<float>(ws, L.A0), at<float>(ws, L.V0), at<float>(ws, L.qbuf), at<double>(ws, L.acc), at<int32_t>(ws, L.order), components_out, variances_out,
                                &sweeps, s);
  if (sweeps_out) *sweeps_out = sweeps;
  if (rc != HME_OK) return rc;
  HME_CUDA(cudaMemcpyAsync(mean_out, at<float>(ws, L.mean32), (size_t)d * 4, cudaMemcpyDeviceToDevice, s),
           "pca: copy mean");
  return HME_OK;
}

int hme_pca_transform(const void *X, int64_t N, int32_t d, int64_t ldx, int32_t dtype, const float *mean,
                      const float *components, int32_t r, float *Z_out, int64_t ldz, void *ws, size_t ws_bytes,
                      void *stream) {
  HME_TRY(check_pca(X, N, d, ldx, dtype, r, 0));
  if (r > kMaxBN) return fail(HME_EINVAL, "r = %d: hme_pca_transform takes at most %d components", r, kMaxBN);
  if (!mean || !components) return fail(HME_EINVAL, "mean / components is NULL");
  if (N > 0 && !Z_out) return fail(HME_EINVAL, "Z_out is NULL");
  if (ldz < r) return fail(HME_EINVAL, "ldz = %lld < r = %d", (long long)ldz, r);
  const AssignGeom g = assign_geom(d, r, HME_F32);
  if (N > 0 && !split_eligible(X, ldx, g))
    return fail(HME_EINVAL, "X must start on a 16-byte boundary with ldx %% 4 == 0 (TMA)");
  const PcaTLayout L = pca_t_layout(d, r);
  HME_TRY(check_ws(ws, ws_bytes, L.total));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  HME_TRY(clear_header(ws, s));
  if (N == 0) return HME_OK;
  Header *hdr = at<Header>(ws, 0);
  HME_CUDA(launch_prep_centres(components, g, at<__nv_bfloat16>(ws, L.chi), at<__nv_bfloat16>(ws, L.clo),
                               at<float>(ws, L.cn), hdr, s),
           "pca: prepare components");
  HME_CUDA(launch_pca_zoff(mean, components, d, r, g.Kp, at<float>(ws, L.zoff), s), "pca: offsets");
  SplitOut out;
  out.z = Z_out;
  out.ldz = ldz;
  out.zcols = r;
  HME_TRY(launch_assign_split(static_cast<const float *>(X), N, ldx, g, at<__nv_bfloat16>(ws, L.chi),
                              at<__nv_bfloat16>(ws, L.clo), at<float>(ws, L.zoff), nullptr, nullptr, hdr, nullptr,
                              nullptr, out, s));
  return HME_OK;
}

int hme_kmeans_stream(const void *X, int64_t N, int32_t d, int64_t ldx, int32_t dtype, int32_t K, int32_t iters,
                      int64_t chunk_rows, float *C_inout, int32_t *labels_out, float *mind_out,
                      double *objectives_out, int64_t *counts_out, int32_t *n_reseeded_out, void *ws, size_t ws_bytes,
                      void *stream) {
  HME_TRY(check_common(N, d, K, dtype));
  if (N < 1) return fail(HME_EINVAL, "N = %lld: nothing to cluster", (long long)N);
  if (iters < 0) return fail(HME_EINVAL, "iters = %d is negative", iters);
  if (chunk_rows < 1) return fail(HME_EINVAL, "chunk_rows = %lld must be positive", (long long)chunk_rows);
  if (!X || !C_inout || !labels_out || !mind_out) return fail(HME_EINVAL, "X / C_inout / labels_out / mind_out is NULL");
  if (ldx < d) return fail(HME_EINVAL, "ldx = %lld < d = %d", (long long)ldx, d);
  const int64_t chunk = chunk_rows < N ? chunk_rows : N;
  // X is read by the copy engine; the re-seed reads its picked rows in place,
  // so host memory must be page-locked (device-accessible).
  cudaPointerAttributes attr;
  HME_CUDA(cudaPointerGetAttributes(&attr, X), "query X");
  const void *Xdev = nullptr;
  if (attr.type == cudaMemoryTypeDevice || attr.type == cudaMemoryTypeManaged)
    Xdev = X;
  else if (attr.type == cudaMemoryTypeHost)
    Xdev = attr.devicePointer;
  if (!Xdev) return fail(HME_EINVAL, "X must be page-locked host memory or device memory");
  if (ws_bytes < stream_ws_bytes(chunk, d, K, dtype))
    return fail(HME_ENOMEM, "workspace of %zu bytes is smaller than the %zu bytes needed", ws_bytes,
                stream_ws_bytes(chunk, d, K, dtype));
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return fail(HME_EINVAL, "workspace is NULL or not 256-byte aligned");
  const Layout L = feature_layout(chunk, d, K, dtype, 0);
  const size_t e = dtype == HME_F32 ? 4 : 2;
  const int64_t ldc = stream_ld(d, dtype);
  char *buf[2] = {static_cast<char *>(ws) + align_up(L.total, 256),
                  static_cast<char *>(ws) + align_up(L.total, 256) + stream_buf_bytes(chunk, d, dtype)};
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  HME_TRY(clear_header(ws, s));
  Header *hdr = at<Header>(ws, 0);
  int64_t *hist = at<int64_t>(ws, L.part.hist);
  int64_t *offs = at<int64_t>(ws, L.part.offs);
  int32_t *perm = at<int32_t>(ws, L.perm);
  int32_t *slab = at<int32_t>(ws, L.slab);
  UpdateState st{at<double>(ws, L.sums), at<int64_t>(ws, L.counts), at<double>(ws, L.x2sum)};
  int32_t *dk = at<int32_t>(ws, L.delta_k);
  int32_t *fl = at<int32_t>(ws, L.flagged);
  DeltaScratch ds{dk, dk + K, dk + 2 * K, dk + 3 * K, reinterpret_cast<int64_t *>(dk + 4 * K),
                  perm, slab, fl, fl + chunk, at<unsigned long long>(ws, L.reseed), at<int32_t>(ws, L.delta_mat)};

  // copies of chunk j + 1 run on their own stream while chunk j is clustered
  cudaStream_t cs = nullptr;
  cudaEvent_t ready[2] = {nullptr, nullptr}, done[2] = {nullptr, nullptr};
  int rc = HME_OK;
  auto cuda_ok = [&](cudaError_t err, const char *what) {
    if (err != cudaSuccess && rc == HME_OK) rc = cuda_fail(err, what);
    return rc == HME_OK;
  };
  if (cuda_ok(cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking), "stream: copy stream"))
    for (int b = 0; b < 2 && rc == HME_OK; ++b) {
      cuda_ok(cudaEventCreateWithFlags(&ready[b], cudaEventDisableTiming), "stream: event");
      if (rc == HME_OK) cuda_ok(cudaEventCreateWithFlags(&done[b], cudaEventDisableTiming), "stream: event");
      if (rc == HME_OK) cuda_ok(cudaEventRecord(done[b], s), "stream: event");
    }
  const int64_t nchunks = (N + chunk - 1) / chunk;
  for (int t = 0; t < iters && rc == HME_OK; ++t) {
    for (int64_t j = 0; j < nchunks && rc == HME_OK; ++j) {
      const int64_t r0 = j * chunk, n = (N - r0) < chunk ? (N - r0) : chunk;
      const int b = (int)(j & 1);
      if (!cuda_ok(cudaStreamWaitEvent(cs, done[b], 0), "stream: wait buffer")) break;
      const char *src = static_cast<const char *>(X) + (size_t)r0 * ldx * e;
      const cudaError_t ce =
          ldx == ldc ? cudaMemcpyAsync(buf[b], src, (size_t)n * ldc * e, cudaMemcpyDefault, cs)  // contiguous rows
                     : cudaMemcpy2DAsync(buf[b], (size_t)ldc * e, src, (size_t)ldx * e, (size_t)d * e, (size_t)n,
                                         cudaMemcpyDefault, cs);
      if (!cuda_ok(ce, "stream: copy chunk")) break;
      if (!cuda_ok(cudaEventRecord(ready[b], cs), "stream: event")) break;
      if (!cuda_ok(cudaStreamWaitEvent(s, ready[b], 0), "stream: wait chunk")) break;
      // this chunk's re-score queues and centre-norm maximum start at zero
      if (!cuda_ok(cudaMemsetAsync(&hdr->rescore_count, 0, 3 * sizeof(uint32_t), s), "stream: clear queues")) break;
      if (!cuda_ok(cudaMemsetAsync(&hdr->cn_max_bits, 0, sizeof(uint32_t), s), "stream: clear queues")) break;
      rc = do_assign(buf[b], n, d, ldc, dtype, C_inout, K, labels_out + r0, mind_out + r0, L, ws, 0, s);
      if (rc != HME_OK) break;
      if (!cuda_ok(launch_partition(labels_out + r0, n, K, L.part, static_cast<char *>(ws), hist, offs, perm, slab,
                                    hdr, s),
                   "stream: sort labels"))
        break;
      if (!cuda_ok(launch_update_add(buf[b], n, d, ldc, dtype, perm, slab, hist, offs + K, K, st, j == 0, s),
                   "stream: sums"))
        break;
      cuda_ok(cudaEventRecord(done[b], s), "stream: event");
    }
    if (rc != HME_OK) break;
    // objective of (C_t, labels), new centres, re-seeds (picked rows read from X in place)
    if (!cuda_ok(cudaMemsetAsync(&hdr->objective, 0, sizeof(double), s), "stream: clear objective")) break;
    if (!cuda_ok(launch_update_finish(Xdev, N, d, ldx, dtype, mind_out, K, st, ds, C_inout, counts_out,
                                      n_reseeded_out, hdr, s),
                 "stream: centres"))
      break;
    if (objectives_out)
      cuda_ok(cudaMemcpyAsync(objectives_out + t, &hdr->objective, sizeof(double), cudaMemcpyDeviceToDevice, s),
              "stream: copy objective");
  }
  // the copy stream's last work is ordered before the caller's stream goes on
  for (int b = 0; b < 2; ++b)
    if (ready[b]) cudaStreamWaitEvent(s, ready[b], 0);
  for (int b = 0; b < 2; ++b) {
    if (ready[b]) cudaEventDestroy(ready[b]);
    if (done[b]) cudaEventDestroy(done[b]);
  }
  if (cs) cudaStreamDestroy(cs);
  return rc;
}

int hme_debug_bounded_wait(uint64_t timeout_ns, void *ws, size_t ws_bytes, void *stream) {
  if (timeout_ns < 1 || timeout_ns > 1000000000ull) return fail(HME_EINVAL, "timeout_ns out of range");
  HME_TRY(check_ws(ws, ws_bytes, sizeof(Header)));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  HME_TRY(clear_header(ws, s));
  HME_CUDA(launch_debug_wait(timeout_ns, at<Header>(ws, 0), s), "debug wait");
  return HME_OK;
}

}  // extern "C"
