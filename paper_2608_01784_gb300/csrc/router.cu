// router.cu — router scores, variable-count TopK and normalised router
// weights of the token-choice MoE layer (REFLEX Sec. 3.2, Eq. 2).
//
// Scores.  z[t, e] = sum_k h[t, k] * W_r[e, k] is evaluated, for every
// (t, e), as the sequential chain acc = fma(h[t,k], W_r[e,k], acc) over
// k = 0, 1, ..., d-1 starting from +0, in fp32 (bf16 inputs are widened
// exactly).  Fixing the summation order makes the scores — and therefore the
// selected expert sets, an integer result — reproducible bit for bit.  The
// kernel is a register-tiled SIMT GEMM: each thread owns TM tokens x 4
// experts and walks k in order, so the fixed order costs no extra work; the
// tile (8*TM tokens x 64 experts) is staged through double-buffered shared
// memory in chunks of 32 k.
//
// Selection.  One warp per token keeps E/32 scores per lane and runs k_i
// rounds of a warp-wide max over packed 64-bit keys
//   key = (order-preserving bits of z) << 32 | (0xffffffff - e)
// so the larger score wins and, on equal scores, the lower expert index.
// alpha is the softmax weight, renormalised over the selected set by default.
#include "common.cuh"
#include "internal.h"

namespace rx {
namespace {

constexpr int kKc = 32;          // k per shared-memory chunk
constexpr int kExpPerCta = 64;   // 16 thread columns x 4 experts
constexpr int kThreadsL = 128;   // 16 x 8 threads

template <typename Tin, int TM>
__global__ void __launch_bounds__(kThreadsL)
    logits_kernel(const Tin* __restrict__ h, const Tin* __restrict__ w, int T,
                  int d, int E, float* __restrict__ z) {
  constexpr int BT = 8 * TM;  // tokens per CTA
  __shared__ __align__(16) float hs[2][kKc][BT];
  __shared__ __align__(16) float ws[2][kKc][kExpPerCta];
  const int tx = threadIdx.x & 15;  // expert group (4 experts)
  const int ty = threadIdx.x >> 4;  // token group (TM tokens)
  const int t0 = blockIdx.x * BT;
  const int e0 = blockIdx.y * kExpPerCta;

  // loader: h tile = BT rows x 4 vectors of 8; w tile = 64 rows x 4 vectors
  constexpr int kHVec = BT * (kKc / 8);
  float hv[8], wv[2][8];
  const int nchunks = d / kKc;

  auto load_regs = [&](int c) {
    const int k0 = c * kKc;
    if (threadIdx.x < kHVec) {
      const int r = threadIdx.x >> 2, v = threadIdx.x & 3;
      const int t = t0 + r;
      if (t < T) {
        load8(h + static_cast<int64_t>(t) * d + k0 + v * 8, hv);
      } else {
#pragma unroll
        for (int i = 0; i < 8; ++i) hv[i] = 0.f;
      }
    }
#pragma unroll
    for (int s = 0; s < 2; ++s) {
      const int idx = threadIdx.x + s * kThreadsL;
      const int r = idx >> 2, v = idx & 3;
      const int e = e0 + r;
      if (e < E) {
        load8(w + static_cast<int64_t>(e) * d + k0 + v * 8, wv[s]);
      } else {
#pragma unroll
        for (int i = 0; i < 8; ++i) wv[s][i] = 0.f;
      }
    }
  };
  auto store_smem = [&](int buf) {
    if (threadIdx.x < kHVec) {
      const int r = threadIdx.x >> 2, v = threadIdx.x & 3;
#pragma unroll
      for (int i = 0; i < 8; ++i) hs[buf][v * 8 + i][r] = hv[i];
    }
#pragma unroll
    for (int s = 0; s < 2; ++s) {
      const int idx = threadIdx.x + s * kThreadsL;
      const int r = idx >> 2, v = idx & 3;
#pragma unroll
      for (int i = 0; i < 8; ++i) ws[buf][v * 8 + i][r] = wv[s][i];
    }
  };

  float acc[TM][4];
#pragma unroll
  for (int i = 0; i < TM; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

  load_regs(0);
  store_smem(0);
  __syncthreads();
  for (int c = 0; c < nchunks; ++c) {
    const int buf = c & 1;
    if (c + 1 < nchunks) load_regs(c + 1);
#pragma unroll 8
    for (int kk = 0; kk < kKc; ++kk) {
      const float4 wq = *reinterpret_cast<const float4*>(&ws[buf][kk][tx * 4]);
      float hq[TM];
      if constexpr (TM == 4) {
        const float4 t4 = *reinterpret_cast<const float4*>(&hs[buf][kk][ty * 4]);
        hq[0] = t4.x; hq[1] = t4.y; hq[2] = t4.z; hq[3] = t4.w;
      } else if constexpr (TM == 2) {
        const float2 t2 = *reinterpret_cast<const float2*>(&hs[buf][kk][ty * 2]);
        hq[0] = t2.x; hq[1] = t2.y;
      } else {
        hq[0] = hs[buf][kk][ty];
      }
#pragma unroll
      for (int i = 0; i < TM; ++i) {
        acc[i][0] = __fmaf_rn(hq[i], wq.x, acc[i][0]);
        acc[i][1] = __fmaf_rn(hq[i], wq.y, acc[i][1]);
        acc[i][2] = __fmaf_rn(hq[i], wq.z, acc[i][2]);
        acc[i][3] = __fmaf_rn(hq[i], wq.w, acc[i][3]);
      }
    }
    if (c + 1 < nchunks) store_smem(buf ^ 1);
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < TM; ++i) {
    const int t = t0 + ty * TM + i;
    if (t >= T) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int e = e0 + tx * 4 + j;
      if (e < E) z[static_cast<int64_t>(t) * E + e] = acc[i][j];
    }
  }
}

__device__ __forceinline__ uint32_t order_bits(float v) {
  const uint32_t u = __float_as_uint(v);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float from_order_bits(uint32_t o) {
  return __uint_as_float((o & 0x80000000u) ? (o & 0x7fffffffu) : ~o);
}

constexpr int kSelWarps = 8;

template <int NPL>
__global__ void __launch_bounds__(kSelWarps * 32)
    select_kernel(const float* __restrict__ z, const int32_t* __restrict__ kin,
                  int T, int E, int k_max, int renorm,
                  int32_t* __restrict__ ids, float* __restrict__ alpha,
                  uint32_t* __restrict__ err) {
  __shared__ float s_z[kSelWarps][32];
  __shared__ int32_t s_e[kSelWarps][32];
  const int wid = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t = blockIdx.x * kSelWarps + wid;
  if (t >= T) return;
  const int kcap = k_max < E ? k_max : E;
  int kt = kin[t];
  if (kt < 1 || kt > kcap) {
    if (lane == 0) set_err(err, kErrKRange);
    kt = kt < 1 ? 1 : kcap;
  }
  float zv[NPL];
  unsigned long long key[NPL];
  const float* zt = z + static_cast<int64_t>(t) * E;
#pragma unroll
  for (int i = 0; i < NPL; ++i) {
    const int e = lane + 32 * i;
    if (e < E) {
      float v = zt[e];
      v = (v == 0.0f) ? 0.0f : v;  // -0 and +0 are equal scores
      zv[i] = v;
      key[i] = (static_cast<unsigned long long>(order_bits(v)) << 32) |
               static_cast<unsigned long long>(0xffffffffu - static_cast<uint32_t>(e));
    } else {
      zv[i] = -INFINITY;
      key[i] = 0ull;
    }
  }
  for (int j = 0; j < kt; ++j) {
    unsigned long long best = key[0];
#pragma unroll
    for (int i = 1; i < NPL; ++i) best = key[i] > best ? key[i] : best;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const unsigned long long other = __shfl_xor_sync(0xffffffffu, best, o);
      best = other > best ? other : best;
    }
    const int e = static_cast<int>(0xffffffffu - static_cast<uint32_t>(best & 0xffffffffull));
    if ((e & 31) == lane) {
#pragma unroll
      for (int i = 0; i < NPL; ++i)
        if (i == (e >> 5)) key[i] = 0ull;
    }
    if (lane == 0) {
      s_e[wid][j] = e;
      s_z[wid][j] = from_order_bits(static_cast<uint32_t>(best >> 32));
    }
  }
  __syncwarp();
  const float zmax = s_z[wid][0];
  float all = 0.f;
#pragma unroll
  for (int i = 0; i < NPL; ++i)
    if (lane + 32 * i < E) all += expf(zv[i] - zmax);
  const float mine = lane < kt ? expf(s_z[wid][lane] - zmax) : 0.f;
  float sel = mine;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    all += __shfl_xor_sync(0xffffffffu, all, o);
    sel += __shfl_xor_sync(0xffffffffu, sel, o);
  }
  const float denom = renorm ? sel : all;
  for (int j = lane; j < k_max; j += 32) {
    const int64_t o = static_cast<int64_t>(t) * k_max + j;
    if (j < kt) {
      ids[o] = s_e[wid][j];
      alpha[o] = mine / denom;
    } else {
      ids[o] = -1;
      alpha[o] = 0.f;
    }
  }
}

template <typename Tin>
cudaError_t logits_dispatch(const Tin* h, const Tin* w, int T, int d, int E,
                            float* z, int num_sms, cudaStream_t s) {
  const int gy = (E + kExpPerCta - 1) / kExpPerCta;
  auto grid_for = [&](int tm) { return ((T + 8 * tm - 1) / (8 * tm)) * gy; };
  const int want = 2 * num_sms;
  if (grid_for(4) >= want) {
    dim3 g((T + 31) / 32, gy);
    logits_kernel<Tin, 4><<<g, kThreadsL, 0, s>>>(h, w, T, d, E, z);
  } else if (grid_for(2) >= want) {
    dim3 g((T + 15) / 16, gy);
    logits_kernel<Tin, 2><<<g, kThreadsL, 0, s>>>(h, w, T, d, E, z);
  } else {
    dim3 g((T + 7) / 8, gy);
    logits_kernel<Tin, 1><<<g, kThreadsL, 0, s>>>(h, w, T, d, E, z);
  }
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_router_logits(int dtype, const void* hidden,
                                 const void* w_router, int T, int d, int E,
                                 float* z, int num_sms, cudaStream_t stream) {
  if (T == 0) return cudaSuccess;
  if (dtype == 0)
    return logits_dispatch(static_cast<const float*>(hidden),
                           static_cast<const float*>(w_router), T, d, E, z,
                           num_sms, stream);
  return logits_dispatch(static_cast<const __nv_bfloat16*>(hidden),
                         static_cast<const __nv_bfloat16*>(w_router), T, d, E,
                         z, num_sms, stream);
}

cudaError_t launch_router_select(const float* z, const int32_t* k, int T,
                                 int E, int k_max, bool renorm, int32_t* ids,
                                 float* alpha, uint32_t* err,
                                 cudaStream_t stream) {
  if (T == 0) return cudaSuccess;
  const dim3 grid((T + kSelWarps - 1) / kSelWarps);
  const dim3 block(kSelWarps * 32);
  const int r = renorm ? 1 : 0;
  if (E <= 32)
    select_kernel<1><<<grid, block, 0, stream>>>(z, k, T, E, k_max, r, ids, alpha, err);
  else if (E <= 64)
    select_kernel<2><<<grid, block, 0, stream>>>(z, k, T, E, k_max, r, ids, alpha, err);
  else if (E <= 128)
    select_kernel<4><<<grid, block, 0, stream>>>(z, k, T, E, k_max, r, ids, alpha, err);
  else if (E <= 256)
    select_kernel<8><<<grid, block, 0, stream>>>(z, k, T, E, k_max, r, ids, alpha, err);
  else if (E <= 512)
    select_kernel<16><<<grid, block, 0, stream>>>(z, k, T, E, k_max, r, ids, alpha, err);
  else
    select_kernel<32><<<grid, block, 0, stream>>>(z, k, T, E, k_max, r, ids, alpha, err);
  return cudaGetLastError();
}

}  // namespace rx
