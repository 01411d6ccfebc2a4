// combine.cu — the weighted sum of Eq. 2 (REFLEX Sec. 3.2) back in token
// order: out_t = sum_{j < k_t} alpha[t, j] * y[row_of[t, j]] (+ shared_t)
// (+ resid_t, the layer input, for stacked layers).
//
// Each thread owns 8 consecutive columns of one token (d / 8 threads per
// token, 256 threads per CTA), so every load and store is one 16-byte (bf16)
// or 32-byte (fp32) vector and a token's row is read by consecutive threads.
// The CTAs are persistent (a few per SM) and walk the tokens in groups; the
// pair rows, weights and count of the next group are copied into shared
// memory with cp.async while the current group is summed, so each token costs
// one round trip per 4 slots (their rows loaded back to back) instead of
// a chain of metadata loads, barriers and row loads.  Sums are fp32 in slot
// order j = 0, 1, ..., then rounded once to the output type.
#include "common.cuh"
#include "internal.h"

namespace rx {
namespace {

constexpr int kThreads = 256;
constexpr int kMaxK = 32;
constexpr int kBatch = 4;        // slots whose rows are loaded back to back
constexpr int kCtasPerSm = 6;

// 8 raw elements: loaded as stored, widened exactly to fp32 when summed.
template <typename Te>
struct Raw8;
template <>
struct Raw8<__nv_bfloat16> {
  uint4 v;
  __device__ __forceinline__ void load(const __nv_bfloat16* p) {
    v = *reinterpret_cast<const uint4*>(p);
  }
  __device__ __forceinline__ void zero() { v = make_uint4(0u, 0u, 0u, 0u); }
  __device__ __forceinline__ void widen(float* f) const {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      f[2 * i] = __uint_as_float(w[i] << 16);
      f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
    }
  }
};
template <>
struct Raw8<float> {
  float4 a, b;
  __device__ __forceinline__ void load(const float* p) {
    a = *reinterpret_cast<const float4*>(p);
    b = *reinterpret_cast<const float4*>(p + 4);
  }
  __device__ __forceinline__ void zero() { a = b = make_float4(0.f, 0.f, 0.f, 0.f); }
  __device__ __forceinline__ void widen(float* f) const {
    f[0] = a.x; f[1] = a.y; f[2] = a.z; f[3] = a.w;
    f[4] = b.x; f[5] = b.y; f[6] = b.z; f[7] = b.w;
  }
};

__device__ __forceinline__ void cp_async4(void* smem, const void* gmem) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_addr(smem)),
               "l"(gmem)
               : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.wait_all;" ::: "memory");
}

template <typename Te>
__global__ void __launch_bounds__(kThreads)
    combine_kernel(const Te* __restrict__ y, const Te* __restrict__ ysh,
                   const Te* __restrict__ resid, const int32_t* __restrict__ row_of,
                   const float* __restrict__ alpha, const int32_t* __restrict__ k,
                   int T, int d, int k_max, int cap_rows, Te* __restrict__ out,
                   uint32_t* __restrict__ err) {
  const int tpt = d / 8;                 // threads per token (d <= 2048)
  const int tpc = kThreads / tpt;        // tokens per group
  const int sub = threadIdx.x / tpt;     // token slot within the group
  const int lt = threadIdx.x % tpt;
  const int c = lt * 8;
  __shared__ int32_t s_row[2][kThreads / 8][kMaxK];
  __shared__ float s_a[2][kThreads / 8][kMaxK];
  __shared__ int32_t s_k[2][kThreads / 8];
  grid_dep_wait();
  grid_dep_launch();
  const int ngroups = (T + tpc - 1) / tpc;
  // the metadata of group g into buffer buf: k_max rows and weights per token
  auto prefetch = [&](int g, int buf) {
    const int n = tpc * k_max;
    for (int i = threadIdx.x; i < 2 * n + tpc; i += kThreads) {
      if (i < 2 * n) {
        const int ii = i < n ? i : i - n;
        const int sl = ii / k_max, j = ii % k_max;
        const int t = g * tpc + sl;
        if (t >= T) continue;
        const int64_t o = static_cast<int64_t>(t) * k_max + j;
        if (i < n)
          cp_async4(&s_row[buf][sl][j], row_of + o);
        else
          cp_async4(&s_a[buf][sl][j], alpha + o);
      } else {
        const int sl = i - 2 * n;
        const int t = g * tpc + sl;
        if (t < T) cp_async4(&s_k[buf][sl], k + t);
      }
    }
  };
  int buf = 0;
  if (blockIdx.x < ngroups) prefetch(blockIdx.x, 0);
  cp_async_wait_all();
  __syncthreads();
  for (int g = blockIdx.x; g < ngroups; g += gridDim.x, buf ^= 1) {
    if (g + gridDim.x < ngroups) prefetch(g + gridDim.x, buf ^ 1);
    const int t = g * tpc + sub;
    if (sub < tpc && t < T) {
      int kt = s_k[buf][sub];
      kt = kt < 1 ? 1 : (kt > k_max ? k_max : kt);
      float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
      for (int j0 = 0; j0 < kt; j0 += kBatch) {
        Raw8<Te> v[kBatch];
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
          const int j = j0 + u;
          int r = j < kt ? s_row[buf][sub][j] : -1;
          // -1 marks a slot the router clamped away (already flagged there)
          if (r >= cap_rows) {
            if (lt == 0) set_err(err, kErrIndex);
            r = -1;
          }
          if (r >= 0)
            v[u].load(y + static_cast<int64_t>(r) * d + c);
          else
            v[u].zero();
        }
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
          const int j = j0 + u;
          if (j < kt) {
            const float a = s_a[buf][sub][j];
            float f[8];
            v[u].widen(f);
#pragma unroll
            for (int i = 0; i < 8; ++i) acc[i] = __fmaf_rn(a, f[i], acc[i]);
          }
        }
      }
      if (ysh != nullptr) {
        float f[8];
        load8(ysh + static_cast<int64_t>(t) * d + c, f);
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[i] += f[i];
      }
      if (resid != nullptr) {
        float f[8];
        load8(resid + static_cast<int64_t>(t) * d + c, f);
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[i] += f[i];
      }
      store8(out + static_cast<int64_t>(t) * d + c, acc);
    }
    cp_async_wait_all();  // the next group's metadata has landed
    __syncthreads();      // ... for every thread; this group's buffer is free
  }
}

// d > 2048: one warp per token, 256-column passes.
template <typename Te>
__global__ void __launch_bounds__(kThreads)
    combine_wide_kernel(const Te* __restrict__ y, const Te* __restrict__ ysh,
                        const Te* __restrict__ resid, const int32_t* __restrict__ row_of,
                        const float* __restrict__ alpha,
                        const int32_t* __restrict__ k, int T, int d, int k_max,
                        int cap_rows, Te* __restrict__ out,
                        uint32_t* __restrict__ err) {
  grid_dep_wait();
  grid_dep_launch();
  const int lane = threadIdx.x & 31;
  const int t = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (t >= T) return;
  int kt = k[t];
  kt = kt < 1 ? 1 : (kt > k_max ? k_max : kt);
  int my_row = -1;
  float my_a = 0.f;
  if (lane < kt) {
    my_row = row_of[static_cast<int64_t>(t) * k_max + lane];
    my_a = alpha[static_cast<int64_t>(t) * k_max + lane];
    if (my_row >= cap_rows) set_err(err, kErrIndex);
    if (my_row < 0 || my_row >= cap_rows) my_row = -1;
  }
  for (int c = lane * 8; c < d; c += 256) {
    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    for (int j = 0; j < kt; ++j) {
      const int r = __shfl_sync(0xffffffffu, my_row, j);
      const float a = __shfl_sync(0xffffffffu, my_a, j);
      if (r < 0) continue;
      float v[8];
      load8(y + static_cast<int64_t>(r) * d + c, v);
#pragma unroll
      for (int i = 0; i < 8; ++i) acc[i] = __fmaf_rn(a, v[i], acc[i]);
    }
    if (ysh != nullptr) {
      float v[8];
      load8(ysh + static_cast<int64_t>(t) * d + c, v);
#pragma unroll
      for (int i = 0; i < 8; ++i) acc[i] += v[i];
    }
    if (resid != nullptr) {
      float v[8];
      load8(resid + static_cast<int64_t>(t) * d + c, v);
#pragma unroll
      for (int i = 0; i < 8; ++i) acc[i] += v[i];
    }
    store8(out + static_cast<int64_t>(t) * d + c, acc);
  }
}

template <typename Te>
cudaError_t launch_typed(const Te* y, const Te* ysh, const Te* resid, const int32_t* row_of,
                         const float* alpha, const int32_t* k, int T, int d,
                         int k_max, int cap_rows, Te* out, uint32_t* err, int num_sms,
                         cudaStream_t stream) {
  if (d <= 2048 && kThreads % (d / 8) == 0 && k_max <= kMaxK) {
    const int tok_per_cta = kThreads / (d / 8);
    const int groups = (T + tok_per_cta - 1) / tok_per_cta;
    const int cap = kCtasPerSm * (num_sms > 0 ? num_sms : 1);
    const int grid = groups < cap ? groups : cap;
    return launch_pdl(combine_kernel<Te>, dim3(grid), dim3(kThreads), 0, stream, y, ysh, resid,
                      row_of, alpha, k, T, d, k_max, cap_rows, out, err);
  }
  return launch_pdl(combine_wide_kernel<Te>, dim3((T + 7) / 8), dim3(kThreads), 0, stream, y,
                    ysh, resid, row_of, alpha, k, T, d, k_max, cap_rows, out, err);
}

}  // namespace

cudaError_t launch_combine(int dtype, const void* y, const void* y_shared,
                           const void* resid, const int32_t* row_of, const float* alpha,
                           const int32_t* k, int T, int d, int k_max,
                           int cap_rows, void* out, uint32_t* err, int num_sms,
                           cudaStream_t stream) {
  if (T == 0) return cudaSuccess;
  if (dtype == 0)
    return launch_typed(static_cast<const float*>(y),
                        static_cast<const float*>(y_shared),
                        static_cast<const float*>(resid), row_of, alpha, k, T,
                        d, k_max, cap_rows, static_cast<float*>(out), err, num_sms, stream);
  return launch_typed(static_cast<const __nv_bfloat16*>(y),
                      static_cast<const __nv_bfloat16*>(y_shared),
                      static_cast<const __nv_bfloat16*>(resid), row_of, alpha,
                      k, T, d, k_max, cap_rows, static_cast<__nv_bfloat16*>(out),
                      err, num_sms, stream);
}

}  // namespace rx
