// common.cuh — shared internals of the REFLEX GB300 path (device error bits,
// workspace header, element helpers, bounded mbarrier waits).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace rx {

// Device error word bits (OR-ed by kernels, mapped to REFLEX_* on the host).
constexpr uint32_t kErrKRange = 1u;    // a count outside [1, min(k_max, E)]
constexpr uint32_t kErrTimeout = 2u;   // a bounded wait expired
constexpr uint32_t kErrCapacity = 4u;  // too many active-block tokens
constexpr uint32_t kErrActive = 8u;    // active block index < 1
constexpr uint32_t kErrIndex = 16u;    // an index read from the workspace was
                                       // out of range (stage run out of order)

// First 256 bytes of every forward workspace.
struct WsHeader {
  uint32_t err;          // device error word
  int32_t total_pairs;   // sum_i k_i after dispatch
  int32_t total_mtiles;  // sum_e ceil(count_e / 128) after dispatch
  int32_t total_mtiles2; // sum_e ceil(count_e / 256) after dispatch
  int32_t pad[60];
};
static_assert(sizeof(WsHeader) == 256, "header is 256 bytes");

constexpr int kTileM = 128;  // rows per grouped-GEMM tile (M of tcgen05.mma)

// ---- programmatic dependent launch -----------------------------------------
// The kernels after the first of a call are launched with programmatic stream
// serialization: the next kernel in the stream may be scheduled while the
// current one drains and runs its prologue (barrier setup, TMEM allocation)
// early.  grid_dep_wait() returns once the preceding kernel has completed and
// its writes are visible; every kernel calls it before its first global
// memory access, so stream order is kept exactly.  grid_dep_launch() allows
// the following kernel to be scheduled.  Both are no-ops for plain launches.
__device__ __forceinline__ void grid_dep_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}
__device__ __forceinline__ void grid_dep_launch() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t stream, Args... args) {
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}

// ---- exp in fp32 from a published method ----------------------------------
// Written from Cody & Waite's argument reduction with a degree-7 Taylor
// polynomial, in separate IEEE operations (no contraction), so every call
// gives the same bits on every launch: the FPS sigmoids of the count kernel
// and the router-mass count rules of the selection take integer decisions
// on it.
__device__ __forceinline__ float pow2i(int e) {  // e in [-126, 127]
  return __int_as_float((e + 127) << 23);
}

// e^x: x = k ln2 + r with k = nearest integer to x / ln2 (ties to even);
// r = (x - k ln2_hi) - k ln2_lo (ln2_hi has 16 significant bits, so k ln2_hi
// is exact); e^r by the Taylor series to r^7 in Horner form; the scale 2^k is
// applied as two powers of two so that neither overflows and a subnormal
// result is rounded once.
__device__ __forceinline__ float exp_cw(float x) {
  if (x != x) return x;
  if (x >= 89.0f) return __int_as_float(0x7f800000);
  if (x <= -104.0f) return 0.0f;
  const float inv_ln2 = 1.44269502162933349609375f;
  const float ln2_hi = 0.693145751953125f;
  const float ln2_lo = 1.428606765330187045037746429443359375e-06f;
  const float kf = rintf(__fmul_rn(x, inv_ln2));
  const int k = static_cast<int>(kf);
  float r = __fsub_rn(x, __fmul_rn(kf, ln2_hi));
  r = __fsub_rn(r, __fmul_rn(kf, ln2_lo));
  float p = 1.98412701138295233249664306640625e-04f;           // 1/7!
  p = __fadd_rn(__fmul_rn(p, r), 1.388888922519981861114501953125e-03f);   // 1/6!
  p = __fadd_rn(__fmul_rn(p, r), 8.333333767950534820556640625e-03f);      // 1/5!
  p = __fadd_rn(__fmul_rn(p, r), 4.16666679084300994873046875e-02f);       // 1/4!
  p = __fadd_rn(__fmul_rn(p, r), 1.6666667163372039794921875e-01f);        // 1/3!
  p = __fadd_rn(__fmul_rn(p, r), 0.5f);
  p = __fadd_rn(__fmul_rn(p, r), 1.0f);
  p = __fadd_rn(__fmul_rn(p, r), 1.0f);
  const int k1 = k >> 1;
  const int k2 = k - k1;
  return __fmul_rn(__fmul_rn(p, pow2i(k1)), pow2i(k2));
}

__device__ __forceinline__ void set_err(uint32_t* err, uint32_t bit) {
  if (err) atomicOr(err, bit);
}

template <typename T>
__device__ __forceinline__ float to_f32(T v);
template <>
__device__ __forceinline__ float to_f32<float>(float v) { return v; }
template <>
__device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 v) {
  return __bfloat162float(v);
}

template <typename T>
__device__ __forceinline__ T from_f32(float v);
template <>
__device__ __forceinline__ float from_f32<float>(float v) { return v; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float v) {
  return __float2bfloat16_rn(v);
}

// 8 consecutive elements <-> 8 floats (16-byte bf16 / 32-byte fp32 vectors).
__device__ __forceinline__ void load8(const __nv_bfloat16* p, float* f) {
  uint4 v = *reinterpret_cast<const uint4*>(p);
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float2 t = __bfloat1622float2(h[i]);
    f[2 * i] = t.x;
    f[2 * i + 1] = t.y;
  }
}
__device__ __forceinline__ void load8(const float* p, float* f) {
  float4 a = *reinterpret_cast<const float4*>(p);
  float4 b = *reinterpret_cast<const float4*>(p + 4);
  f[0] = a.x; f[1] = a.y; f[2] = a.z; f[3] = a.w;
  f[4] = b.x; f[5] = b.y; f[6] = b.z; f[7] = b.w;
}
__device__ __forceinline__ void store8(__nv_bfloat16* p, const float* f) {
  uint4 v;
  __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&v);
#pragma unroll
  for (int i = 0; i < 4; ++i) h[i] = __floats2bfloat162_rn(f[2 * i], f[2 * i + 1]);
  *reinterpret_cast<uint4*>(p) = v;
}
__device__ __forceinline__ void store8(float* p, const float* f) {
  *reinterpret_cast<float4*>(p) = make_float4(f[0], f[1], f[2], f[3]);
  *reinterpret_cast<float4*>(p + 4) = make_float4(f[4], f[5], f[6], f[7]);
}

// ---- mbarrier primitives with a time limit --------------------------------
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)),
               "r"(count)
               : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Waits for the phase with the given parity to complete.  Gives up after
// limit_ns nanoseconds, or early when *abort becomes non-zero; returns
// whether the phase completed.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity,
                                          const volatile int* abort,
                                          uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (abort != nullptr && *abort) return false;
    if (global_ns() - t0 > limit_ns) return false;
  }
}

// Stage hand-off for TMA-fed rings: the byte count a stage expects (the
// arrival of the thread that issues its copies), a plain local arrival, a
// 2D tiled TMA load whose completion is counted on `bar`.
__device__ __forceinline__ void mbar_arrive_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar),
               "r"(bytes)
               : "memory");
}
// Orders this thread's earlier generic-proxy accesses of shared memory with
// later async-proxy (TMA) accesses: a consumer that read a ring stage with
// ordinary loads issues it before releasing the stage to the next TMA fill.
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_local(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void tma_tile_2d(uint32_t dst, const void* map, int c0, int c1,
                                            uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(bar)
      : "memory");
}

}  // namespace rx
