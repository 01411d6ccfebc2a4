// combine.cu — the weighted sum of Eq. 2 (REFLEX Sec. 3.2) back in token
// order: out_t = sum_{j < k_t} alpha[t, j] * y[row_of[t, j]] (+ shared_t).
//
// One warp per token; each lane owns 8 consecutive columns per 256-column
// pass, so every load and store is a 16-byte (bf16) or 32-byte (fp32) vector
// and a warp touches 512 contiguous bytes per row pass.  The k_t pair rows
// and weights are read once per token into lanes and broadcast by shuffle.
// Sums are fp32, slot order j = 0, 1, ..., then rounded once to the output
// type.
#include "common.cuh"
#include "internal.h"

namespace rx {
namespace {

template <typename Te>
__global__ void __launch_bounds__(256)
    combine_kernel(const Te* __restrict__ y, const Te* __restrict__ ysh,
                   const int32_t* __restrict__ row_of,
                   const float* __restrict__ alpha, const int32_t* __restrict__ k,
                   int T, int d, int k_max, int cap_rows, Te* __restrict__ out,
                   uint32_t* __restrict__ err) {
  const int lane = threadIdx.x & 31;
  const int warps = gridDim.x * 8;
  for (int t = blockIdx.x * 8 + (threadIdx.x >> 5); t < T; t += warps) {
    int kt = k[t];
    kt = kt < 1 ? 1 : (kt > k_max ? k_max : kt);
    int my_row = -1;
    float my_a = 0.f;
    if (lane < kt) {
      my_row = row_of[static_cast<int64_t>(t) * k_max + lane];
      my_a = alpha[static_cast<int64_t>(t) * k_max + lane];
      // -1 marks a slot the router clamped away (already flagged there)
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
      store8(out + static_cast<int64_t>(t) * d + c, acc);
    }
  }
}

}  // namespace

cudaError_t launch_combine(int dtype, const void* y, const void* y_shared,
                           const int32_t* row_of, const float* alpha,
                           const int32_t* k, int T, int d, int k_max,
                           int cap_rows, void* out, uint32_t* err, int num_sms,
                           cudaStream_t stream) {
  if (T == 0) return cudaSuccess;
  int grid = (T + 7) / 8;
  if (grid > 8 * num_sms) grid = 8 * num_sms;
  if (dtype == 0)
    combine_kernel<float><<<grid, 256, 0, stream>>>(
        static_cast<const float*>(y), static_cast<const float*>(y_shared),
        row_of, alpha, k, T, d, k_max, cap_rows, static_cast<float*>(out), err);
  else
    combine_kernel<__nv_bfloat16><<<grid, 256, 0, stream>>>(
        static_cast<const __nv_bfloat16*>(y),
        static_cast<const __nv_bfloat16*>(y_shared), row_of, alpha, k, T, d,
        k_max, cap_rows, static_cast<__nv_bfloat16*>(out), err);
  return cudaGetLastError();
}

}  // namespace rx
