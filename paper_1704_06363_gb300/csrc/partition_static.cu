// partition_static.cu -- hme_partition_noalloc: the expert partition for
// callers that cannot allocate device memory.
//
// Some callers cannot hand this library a workspace: a serving loop that must
// not call cudaMalloc/cudaFree on its request path (both can synchronise the
// whole device), or an application whose device memory is entirely owned by
// another framework's pool.  This entry point needs no workspace: its only
// scratch (a status word and the per-tile bucket counts of the stable
// counting sort) lives in a fixed array in device global memory that is part
// of the library image.
//
// - The array is kStaticScratchBytes = 16 MiB.  Every GPU that loads the
//   library holds it until the process exits.
// - Set-up: the first call on each device, with that device current, looks up
//   the array's device address with cudaGetSymbolAddress (host code cannot use
//   the array's name as a device address).  Make that first call before any
//   stream capture.  The address belongs to the device's current CUDA context:
//   it is kept together with that context and looked up again when the
//   context changes (after cudaDeviceReset, for example), so a stale address
//   is never passed to a kernel.
// - Every call shares the array and it keeps the last call's contents: the
//   status word is cleared at the start of each call; the tile counts are fully
//   rewritten.  Calls that overlap on the GPU (different streams, or several
//   host threads) race on the array and must not be issued.
// - Sizes: the tile length grows so that the ntiles x K counts always fit; a
//   size that would still not fit is rejected with HME_EINVAL.
// - No cudaMalloc, cudaFree or allocating library routine is called.
#include "hme_common.cuh"

#include <mutex>

namespace hme {

namespace {

constexpr size_t kStaticScratchBytes = size_t(16) << 20;

static __device__ __align__(256) unsigned char g_partition_scratch[kStaticScratchBytes];

using CtxGetCurrentFn = CUresult (*)(CUcontext *);

std::mutex g_scratch_mu;
struct ScratchAddr {
  CUcontext ctx;
  void *ptr;
};
ScratchAddr g_scratch[64] = {};

CtxGetCurrentFn ctx_get_current_fn() {
  static CtxGetCurrentFn fn = [] {
    void *f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      return reinterpret_cast<CtxGetCurrentFn>(f);
    return static_cast<CtxGetCurrentFn>(nullptr);
  }();
  return fn;
}

}  // namespace

// The calling thread's current CUDA context (NULL if none or unavailable).
void *current_context_handle() {
  CtxGetCurrentFn get = ctx_get_current_fn();
  CUcontext ctx = nullptr;
  if (!get || get(&ctx) != CUDA_SUCCESS) return nullptr;
  return ctx;
}

namespace {

// Device address of g_partition_scratch in the current device's context (set
// up on the first call in that context).
int static_scratch(void **out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "hme_partition_noalloc: cudaGetDevice");
  if (dev < 0 || dev >= 64) return fail(HME_EINTERNAL, "hme_partition_noalloc: device %d out of range", dev);
  CtxGetCurrentFn get = ctx_get_current_fn();
  if (!get) return fail(HME_ECUDA, "hme_partition_noalloc: cuCtxGetCurrent is not available from the driver");
  CUcontext ctx = nullptr;
  if (get(&ctx) != CUDA_SUCCESS) ctx = nullptr;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (!ctx || g_scratch[dev].ctx != ctx || !g_scratch[dev].ptr) {
    // (the lookup also creates and binds the device's primary context when
    // this thread has none yet)
    void *p = nullptr;
    e = cudaGetSymbolAddress(&p, g_partition_scratch);
    if (e != cudaSuccess) return cuda_fail(e, "hme_partition_noalloc: cudaGetSymbolAddress");
    if (get(&ctx) != CUDA_SUCCESS || !ctx) return fail(HME_ECUDA, "hme_partition_noalloc: no current CUDA context");
    g_scratch[dev] = ScratchAddr{ctx, p};
  }
  *out = g_scratch[dev].ptr;
  return HME_OK;
}

}  // namespace
}  // namespace hme

using namespace hme;

extern "C" int hme_partition_noalloc(const int32_t *labels, int64_t N, int32_t K, int64_t *hist_out,
                                     int64_t *offsets_out, int32_t *perm_out, int32_t *sorted_labels_out,
                                     int32_t *status_out, void *stream) {
  if (N < 0 || N > (int64_t)0x7FFFFFFF) return fail(HME_EINVAL, "N = %lld out of range", (long long)N);
  if (K < 1 || K > kMaxK) return fail(HME_EINVAL, "K = %d out of range [1, %d]", K, kMaxK);
  if (!hist_out || !offsets_out) return fail(HME_EINVAL, "hist_out / offsets_out is NULL");
  if (N > 0 && (!labels || !perm_out)) return fail(HME_EINVAL, "labels / perm_out is NULL");

  // Tile counts go right after the 256-byte header; tiles lengthen (in whole
  // sort chunks) until the ntiles x K counts fit.
  PartLayout pl = part_layout(sizeof(Header), N, K);
  const size_t room = kStaticScratchBytes - sizeof(Header);
  const int64_t max_tiles = (int64_t)(room / ((size_t)K * sizeof(int32_t)));
  if (max_tiles < 1) return fail(HME_EINVAL, "K = %d needs more than %zu bytes of static scratch", K, room);
  if (pl.ntiles > max_tiles) {
    int64_t tile = (N + max_tiles - 1) / max_tiles;
    tile = (tile + kPartChunk - 1) / kPartChunk * kPartChunk;
    pl.tile = tile;
    pl.ntiles = (N + tile - 1) / tile;
  }
  pl.tilecnt = sizeof(Header);
  const size_t need = sizeof(Header) + (size_t)pl.ntiles * K * sizeof(int32_t);
  if (need > kStaticScratchBytes)
    return fail(HME_EINVAL, "N = %lld, K = %d needs %zu bytes of static scratch; the maximum is %zu", (long long)N, K,
                need, kStaticScratchBytes);

  void *scratch = nullptr;
  int rc = static_scratch(&scratch);
  if (rc != HME_OK) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  Header *hdr = static_cast<Header *>(scratch);
  cudaError_t e = cudaMemsetAsync(hdr, 0, sizeof(Header), s);  // the status word must start at zero
  if (e != cudaSuccess) return cuda_fail(e, "hme_partition_noalloc: clear status");
  e = launch_partition(labels, N, K, pl, static_cast<char *>(scratch), hist_out, offsets_out, perm_out,
                       sorted_labels_out, hdr, s);
  if (e != cudaSuccess) return cuda_fail(e, "hme_partition_noalloc");
  if (status_out) {
    e = cudaMemcpyAsync(status_out, &hdr->status, sizeof(int32_t), cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return cuda_fail(e, "hme_partition_noalloc: copy status");
  }
  return HME_OK;
}
