// combine.cu — the weighted sum of Eq. 2 (REFLEX Sec. 3.2) back in token
// order: out_t = sum_{j < k_t} alpha[t, j] * y[row_of[t, j]] (+ shared_t)
// (+ resid_t, the layer input, for stacked layers).
//
// Each thread owns 8 consecutive columns of one token (d / 8 threads per
// token, 256 threads per CTA), so every load and store is one 16-byte (bf16)
// or 32-byte (fp32) vector and a token's row is read by consecutive threads.
// The k_t pair rows and weights of the token are staged in shared memory
// once; the row loads of four slots are issued back to back before their
// multiply-adds so their latencies overlap.  Sums are fp32 in slot order
// j = 0, 1, ..., then rounded once to the output type.
#include "common.cuh"
#include "internal.h"

namespace rx {
namespace {

constexpr int kThreads = 256;
constexpr int kMaxK = 32;

template <typename Te>
__global__ void __launch_bounds__(kThreads)
    combine_kernel(const Te* __restrict__ y, const Te* __restrict__ ysh,
                   const Te* __restrict__ resid, const int32_t* __restrict__ row_of,
                   const float* __restrict__ alpha, const int32_t* __restrict__ k,
                   int T, int d, int k_max, int cap_rows, Te* __restrict__ out,
                   uint32_t* __restrict__ err) {
  const int tpt = d / 8;                 // threads per token (d <= 2048)
  const int tok_per_cta = kThreads / tpt;
  const int sub = threadIdx.x / tpt;     // token slot within the CTA
  const int c = (threadIdx.x % tpt) * 8;
  __shared__ int32_t s_row[kThreads / 8][kMaxK];
  __shared__ float s_a[kThreads / 8][kMaxK];
  __shared__ int s_k[kThreads / 8];
  grid_dep_wait();
  grid_dep_launch();
  const int t = blockIdx.x * tok_per_cta + sub;
  const bool active = sub < tok_per_cta && t < T;
  if (active && threadIdx.x % tpt == 0) {
    int kt = k[t];
    kt = kt < 1 ? 1 : (kt > k_max ? k_max : kt);
    s_k[sub] = kt;
  }
  __syncthreads();
  if (active) {
    const int kt = s_k[sub];
    for (int j = threadIdx.x % tpt; j < kt; j += tpt) {
      int r = row_of[static_cast<int64_t>(t) * k_max + j];
      // -1 marks a slot the router clamped away (already flagged there)
      if (r >= cap_rows) set_err(err, kErrIndex);
      if (r < 0 || r >= cap_rows) r = -1;
      s_row[sub][j] = r;
      s_a[sub][j] = alpha[static_cast<int64_t>(t) * k_max + j];
    }
  }
  __syncthreads();
  if (!active) return;
  const int kt = s_k[sub];
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  for (int j0 = 0; j0 < kt; j0 += 4) {
    float v[4][8];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int j = j0 + u;
      const int r = j < kt ? s_row[sub][j] : -1;
      if (r >= 0) {
        load8(y + static_cast<int64_t>(r) * d + c, v[u]);
      } else {
#pragma unroll
        for (int i = 0; i < 8; ++i) v[u][i] = 0.f;
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int j = j0 + u;
      if (j < kt) {
        const float a = s_a[sub][j];
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[i] = __fmaf_rn(a, v[u][i], acc[i]);
      }
    }
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
                         int k_max, int cap_rows, Te* out, uint32_t* err,
                         cudaStream_t stream) {
  if (d <= 2048 && kThreads % (d / 8) == 0) {
    const int tok_per_cta = kThreads / (d / 8);
    const int grid = (T + tok_per_cta - 1) / tok_per_cta;
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
                           int cap_rows, void* out, uint32_t* err, int,
                           cudaStream_t stream) {
  if (T == 0) return cudaSuccess;
  if (dtype == 0)
    return launch_typed(static_cast<const float*>(y),
                        static_cast<const float*>(y_shared),
                        static_cast<const float*>(resid), row_of, alpha, k, T,
                        d, k_max, cap_rows, static_cast<float*>(out), err, stream);
  return launch_typed(static_cast<const __nv_bfloat16*>(y),
                      static_cast<const __nv_bfloat16*>(y_shared),
                      static_cast<const __nv_bfloat16*>(resid), row_of, alpha,
                      k, T, d, k_max, cap_rows, static_cast<__nv_bfloat16*>(out),
                      err, stream);
}

}  // namespace rx
