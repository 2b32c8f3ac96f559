// ordermoe_dispatch_noalloc: the token permutation of ordermoe_dispatch for
// callers that cannot hand the library a device workspace.
//
// Some callers cannot allocate device memory at the point where they run the
// layer: a plugin hosted by an inference server or another framework that
// owns every device allocation through its own fixed pool, or a serving loop
// that has frozen its memory footprint after start-up and may not call
// cudaMalloc (which can also synchronise the device). For them this entry
// point keeps its scratch (the per-chunk expert histogram) in a fixed
// file-scope device array instead of a caller-provided workspace.
//
// The array lives in every GPU's copy of this library for as long as the
// process keeps the library loaded (64 x 1024 int32 = 256 KB per device).
// Its device address is looked up once per device, with that device current,
// on the first call made on the device; make that first call before any
// stream capture. The address is kept for the life of the process: after a
// cudaDeviceReset of a device it is stale, so a process that resets a device
// must not call this entry point on that device again. All calls share the
// one array: two calls whose kernels overlap on the GPU (different streams,
// or different host threads on the same device) race on it. Nothing in it
// needs clearing: every histogram entry a call reads was written earlier in
// the same call.
#include <mutex>

#include "common.cuh"

namespace om {

int dispatch_launch(const int32_t* chosen, const uint16_t* X, int T, int k, int E, int d,
                    int32_t* offsets, int32_t* row_token, int32_t* row_of, uint16_t* X_perm,
                    int32_t* hist, cudaStream_t stream);

size_t dispatch_workspace_bytes(int64_t n, int E);

constexpr int kNoAllocMaxChunks = 1024;  // => at most 262144 (token, slot) entries per call
constexpr int kNoAllocMaxEntries = kDispatchChunk * kNoAllocMaxChunks;
constexpr int64_t kNoAllocHistEntries = kNoAllocMaxChunks * ORDERMOE_MAX_EXPERTS;
// the histogram of the largest call allowed fits the array
static_assert(dispatch_hist_entries(kNoAllocMaxEntries, ORDERMOE_MAX_EXPERTS) <= kNoAllocHistEntries,
              "fixed scratch smaller than the permutation's histogram at the size limit");

static __device__ __align__(256) int32_t g_noalloc_hist[kNoAllocHistEntries];

constexpr int kMaxDevices = 64;
static std::mutex g_noalloc_mu;
static int32_t* g_noalloc_ptr[kMaxDevices] = {};

// Device address of g_noalloc_hist on the current device (looked up once).
static int noalloc_scratch(int32_t** out) {
  int dev = -1;
  OM_CUDA(cudaGetDevice(&dev));
  if (dev < 0 || dev >= kMaxDevices)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "dispatch_noalloc: device ordinal %d >= %d", dev,
                kMaxDevices);
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  if (g_noalloc_ptr[dev] == nullptr) {
    void* p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_hist);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(g_noalloc_hist)");
    g_noalloc_ptr[dev] = static_cast<int32_t*>(p);
  }
  *out = g_noalloc_ptr[dev];
  return ORDERMOE_OK;
}

}  // namespace om

using namespace om;

extern "C" int ordermoe_dispatch_noalloc(const int32_t* chosen_expert, const uint16_t* X, int T,
                                         int k, int E, int d, int32_t* offsets, int32_t* row_token,
                                         int32_t* row_of, uint16_t* X_perm,
                                         ordermoe_stream_t stream) {
  OM_TRACE();
  if (T < 0 || k <= 0 || k > ORDERMOE_MAX_TOPK || E <= 0 || E > ORDERMOE_MAX_EXPERTS)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE,
                "dispatch_noalloc: need T >= 0, 1 <= k <= 8, 1 <= E <= 64");
  if ((int64_t)T * k > kNoAllocMaxEntries)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE,
                "dispatch_noalloc: T*k = %lld exceeds the fixed scratch limit of %d entries; "
                "use ordermoe_dispatch with a workspace",
                (long long)T * k, kNoAllocMaxEntries);
  if (d <= 0 || d % 8 != 0)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "dispatch_noalloc: d must be a positive multiple of 8");
  if (!offsets) return fail(ORDERMOE_ERR_INVALID_ARG, "dispatch_noalloc: null offsets");
  if (T > 0 && (!chosen_expert || !X || !row_token || !row_of || !X_perm))
    return fail(ORDERMOE_ERR_INVALID_ARG, "dispatch_noalloc: null pointer");
  if (T > 0 && (!aligned16(X) || !aligned16(X_perm)))
    return fail(ORDERMOE_ERR_INVALID_ARG, "dispatch_noalloc: X and X_perm must be 16-byte aligned");
  // the scratch this call's permutation uses, as ordermoe_dispatch sizes it
  if (dispatch_workspace_bytes((int64_t)T * k, E) > sizeof(g_noalloc_hist))
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE,
                "dispatch_noalloc: T*k = %lld needs more than the fixed %zu-byte scratch",
                (long long)T * k, sizeof(g_noalloc_hist));
  int32_t* hist = nullptr;
  int rc = noalloc_scratch(&hist);
  if (rc) return rc;
  return dispatch_launch(chosen_expert, X, T, k, E, d, offsets, row_token, row_of, X_perm, hist,
                         stream);
}
