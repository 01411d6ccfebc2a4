// route_noalloc.cu — a routing entry point for callers that cannot allocate
// device memory.
//
// The regular forward needs a caller-provided workspace.  Some callers have
// no way to obtain one: code running inside a host framework that owns the
// device allocator and forbids side allocations, plugins that may only touch
// buffers handed to them, or environments where cudaMalloc is disallowed
// after start-up.  For them, the routing step (router scores, variable-count
// TopK and router weights) is offered here with its only scratch buffer —
// the fp32 score matrix z [T, E] — placed in a fixed-size array that lives in
// the library's own device memory.
//
// Rules of use:
//   - The array holds REFLEX_NOALLOC_MAX_SCORES floats (4 MiB).  Every GPU on
//     which the library is used keeps it until the process exits.
//   - The first call on a device looks up the array's device address (once
//     per device, with that device current).  Make that first call before
//     any stream capture starts.
//   - All calls share the one array and it keeps whatever the last call
//     wrote.  Nothing in it needs to start at zero: each call writes every
//     score it later reads (a score tile whose bounded wait expires writes
//     -inf, never the previous call's values, and flags REFLEX_ETIMEOUT).
//     Calls whose GPU work overlaps in time (for example on two streams at
//     once) race on the array; serialise them.
//   - The caller's status word is cleared with a 4-byte memset in stream
//     order before the kernels, also when T == 0.
#include <mutex>

#include "common.cuh"
#include "internal.h"
#include "reflex.h"

namespace {

static __device__ __align__(256) float g_route_scores[REFLEX_NOALLOC_MAX_SCORES];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
float* g_scores_addr[kMaxDevices] = {nullptr};
int g_sms[kMaxDevices] = {0};

// Device address of the score array and the SM count for the current
// device; looked up on the first call per device.
bool device_setup(float** addr, int* sms) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return false;
  std::lock_guard<std::mutex> lock(g_mu);
  if (g_scores_addr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_route_scores) != cudaSuccess || p == nullptr) return false;
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
      return false;
    g_scores_addr[dev] = static_cast<float*>(p);
    g_sms[dev] = n;
  }
  *addr = g_scores_addr[dev];
  *sms = g_sms[dev];
  return true;
}

}  // namespace

extern "C" int reflex_route_noalloc(int32_t dtype, const void* hidden,
                                    const void* w_router, const int32_t* k,
                                    int32_t T, int32_t d, int32_t E,
                                    int32_t k_max, uint32_t flags,
                                    int32_t* ids_out, float* alpha_out,
                                    int32_t* dev_status, void* stream) {
  if (dtype != REFLEX_DTYPE_F32 && dtype != REFLEX_DTYPE_BF16) return REFLEX_EINVAL;
  if (T < 0 || d <= 0 || d % 64 != 0 || E < 1 || E > 1024) return REFLEX_EINVAL;
  if (k_max < 1 || k_max > 32) return REFLEX_EINVAL;
  if (static_cast<int64_t>(T) * E > REFLEX_NOALLOC_MAX_SCORES) return REFLEX_EWORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  uint32_t* err = reinterpret_cast<uint32_t*>(dev_status);
  if (T == 0) {
    // nothing to route; the status word still reports this call only
    if (err != nullptr && cudaMemsetAsync(err, 0, sizeof(uint32_t), s) != cudaSuccess)
      return REFLEX_ECUDA;
    return REFLEX_OK;
  }
  if (hidden == nullptr || w_router == nullptr || k == nullptr ||
      ids_out == nullptr || alpha_out == nullptr)
    return REFLEX_EINVAL;
  float* z = nullptr;
  int sms = 0;
  if (!device_setup(&z, &sms)) return REFLEX_ECUDA;
  // the status word is cleared in stream order before any kernel of this
  // call can set a bit in it (a 4-byte memset allocates nothing)
  if (err != nullptr && cudaMemsetAsync(err, 0, sizeof(uint32_t), s) != cudaSuccess)
    return REFLEX_ECUDA;
  if (rx::launch_router_logits(dtype, hidden, w_router, T, d, E, z, nullptr, 0, err, sms,
                               s) != cudaSuccess)
    return REFLEX_ECUDA;
  if (rx::launch_router_select(z, k, T, E, k_max, (flags & REFLEX_FLAG_RENORM_TOPK) != 0,
                               ids_out, alpha_out, err, s) != cudaSuccess)
    return REFLEX_ECUDA;
  return REFLEX_OK;
}
