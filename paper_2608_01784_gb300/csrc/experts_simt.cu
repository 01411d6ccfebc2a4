// experts_simt.cu — SwiGLU expert GEMMs over ragged per-expert row groups on
// the SIMT pipes (fp32 path, and a bf16 cross-check of the tensor-core path).
//
// For the pair rows of expert e (rows [offsets[e], offsets[e+1]) of the
// gathered input), Eq. 2's expert E_e is
//   act[r, c] = silu(x_r . Wg[e, c]) * (x_r . Wu[e, c])      c < inter
//   y[r, n]   = act_r . Wd[e, n]                              n < d
// One warp per (row, column); lanes split the reduction index in 8-element
// vectors (coalesced weight rows) and a butterfly adds the 32 partials.
// Accumulation is fp32; act is rounded to the storage type.
#include "common.cuh"
#include "internal.h"

namespace rx {
namespace {

constexpr int kRowsPerCta = 8;   // one warp per row
constexpr int kColsPerCta = 16;  // columns per CTA (loop inside the warp)

__device__ __forceinline__ int group_of(const GroupRows& g, int r) {
  if (g.offsets == nullptr) return 0;
  int lo = 0, hi = g.E;  // offsets[lo] <= r < offsets[hi]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (g.offsets[mid] <= r) lo = mid; else hi = mid;
  }
  return lo;
}

__device__ __forceinline__ int rows_of(const GroupRows& g) {
  if (g.offsets == nullptr) return g.dense_rows;
  const int n = g.totals[0];
  return n < g.cap_rows ? n : g.cap_rows;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

template <typename Te>
__global__ void __launch_bounds__(kRowsPerCta * 32)
    swiglu_simt_kernel(const Te* __restrict__ x, const Te* __restrict__ wgu,
                       int d, int inter, GroupRows g, Te* __restrict__ act) {
  grid_dep_wait();
  grid_dep_launch();
  const int lane = threadIdx.x & 31;
  const int r = blockIdx.x * kRowsPerCta + (threadIdx.x >> 5);
  if (r >= rows_of(g)) return;
  const int e = group_of(g, r);
  const Te* xr = x + static_cast<int64_t>(r) * d;
  const Te* wg_e = wgu + static_cast<int64_t>(e) * 2 * inter * d;
  for (int cc = 0; cc < kColsPerCta; ++cc) {
    const int c = blockIdx.y * kColsPerCta + cc;
    if (c >= inter) break;
    const Te* wg = wg_e + static_cast<int64_t>(c) * d;
    const Te* wu = wg_e + static_cast<int64_t>(inter + c) * d;
    float ga = 0.f, ua = 0.f;
    for (int k = lane * 8; k < d; k += 256) {
      float xv[8], gv[8], uv[8];
      load8(xr + k, xv);
      load8(wg + k, gv);
      load8(wu + k, uv);
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        ga = __fmaf_rn(xv[i], gv[i], ga);
        ua = __fmaf_rn(xv[i], uv[i], ua);
      }
    }
    ga = warp_sum(ga);
    ua = warp_sum(ua);
    if (lane == 0) {
      const float s = ga / (1.0f + expf(-ga));
      act[static_cast<int64_t>(r) * inter + c] = from_f32<Te>(s * ua);
    }
  }
}

template <typename Te>
__global__ void __launch_bounds__(kRowsPerCta * 32)
    down_simt_kernel(const Te* __restrict__ act, const Te* __restrict__ wd,
                     int d, int inter, GroupRows g, Te* __restrict__ y) {
  grid_dep_wait();
  grid_dep_launch();
  const int lane = threadIdx.x & 31;
  const int r = blockIdx.x * kRowsPerCta + (threadIdx.x >> 5);
  if (r >= rows_of(g)) return;
  const int e = group_of(g, r);
  const Te* ar = act + static_cast<int64_t>(r) * inter;
  const Te* wd_e = wd + static_cast<int64_t>(e) * d * inter;
  for (int nn = 0; nn < kColsPerCta; ++nn) {
    const int n = blockIdx.y * kColsPerCta + nn;
    if (n >= d) break;
    const Te* wrow = wd_e + static_cast<int64_t>(n) * inter;
    float acc = 0.f;
    for (int c = lane * 8; c < inter; c += 256) {
      float av[8], wv[8];
      load8(ar + c, av);
      load8(wrow + c, wv);
#pragma unroll
      for (int i = 0; i < 8; ++i) acc = __fmaf_rn(av[i], wv[i], acc);
    }
    acc = warp_sum(acc);
    if (lane == 0) y[static_cast<int64_t>(r) * d + n] = from_f32<Te>(acc);
  }
}

int max_rows(const GroupRows& g) {
  return g.offsets == nullptr ? g.dense_rows : g.cap_rows;
}

}  // namespace

cudaError_t launch_swiglu_simt(int dtype, const void* x, const void* w_gate_up,
                               int d, int inter, const GroupRows& g, void* act,
                               uint32_t*, cudaStream_t stream) {
  const int rows = max_rows(g);
  if (rows == 0) return cudaSuccess;
  const dim3 grid((rows + kRowsPerCta - 1) / kRowsPerCta,
                  (inter + kColsPerCta - 1) / kColsPerCta);
  if (dtype == 0)
    return launch_pdl(swiglu_simt_kernel<float>, grid, dim3(kRowsPerCta * 32), 0, stream,
                      static_cast<const float*>(x), static_cast<const float*>(w_gate_up), d,
                      inter, g, static_cast<float*>(act));
  return launch_pdl(swiglu_simt_kernel<__nv_bfloat16>, grid, dim3(kRowsPerCta * 32), 0, stream,
                    static_cast<const __nv_bfloat16*>(x),
                    static_cast<const __nv_bfloat16*>(w_gate_up), d, inter, g,
                    static_cast<__nv_bfloat16*>(act));
}

cudaError_t launch_down_simt(int dtype, const void* act, const void* w_down,
                             int d, int inter, const GroupRows& g, void* y,
                             uint32_t*, cudaStream_t stream) {
  const int rows = max_rows(g);
  if (rows == 0) return cudaSuccess;
  const dim3 grid((rows + kRowsPerCta - 1) / kRowsPerCta,
                  (d + kColsPerCta - 1) / kColsPerCta);
  if (dtype == 0)
    return launch_pdl(down_simt_kernel<float>, grid, dim3(kRowsPerCta * 32), 0, stream,
                      static_cast<const float*>(act), static_cast<const float*>(w_down), d,
                      inter, g, static_cast<float*>(y));
  return launch_pdl(down_simt_kernel<__nv_bfloat16>, grid, dim3(kRowsPerCta * 32), 0, stream,
                    static_cast<const __nv_bfloat16*>(act),
                    static_cast<const __nv_bfloat16*>(w_down), d, inter, g,
                    static_cast<__nv_bfloat16*>(y));
}

}  // namespace rx
