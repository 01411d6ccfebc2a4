// router.cu — router scores, variable-count TopK and normalised router
// weights of the token-choice MoE layer (REFLEX Sec. 3.2, Eq. 2).
//
// Scores.  z[t, e] = sum_k h[t, k] * W_r[e, k] is evaluated, for every
// (t, e), as the sequential chain acc = fma(h[t,k], W_r[e,k], acc) over
// k = 0, 1, ..., d-1 starting from +0, in fp32 (bf16 inputs are widened
// exactly).  Fixing the summation order makes the scores — and therefore the
// selected expert sets, an integer result — reproducible bit for bit.  The
// kernels are register-tiled SIMT GEMMs: each thread owns TM tokens x TN
// experts and walks k in order, so the fixed order costs no extra work.  Raw
// tiles stream through a cp.async ring; bf16 operands are read straight from
// it into mixed-precision fmas, fp32 operands through a k-major buffer.
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

constexpr int kKc = 32;      // k per pipeline stage
constexpr int kStagesL = 3;  // cp.async ring depth (raw input tiles)

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem, bool valid) {
  const uint32_t dst = smem_addr(smem);
  const int src_bytes = valid ? 16 : 0;  // 0: zero-fill, nothing is read
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst),
               "l"(gmem), "r"(src_bytes)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// 8 raw fp32 elements (the fp32 score kernels; bf16 scores use the mixed-
// precision fma on raw operands).
__device__ __forceinline__ void widen8(const uint8_t* p, float* f, const float*) {
  const float4 a = *reinterpret_cast<const float4*>(p);
  const float4 b = *reinterpret_cast<const float4*>(p + 16);
  f[0] = a.x; f[1] = a.y; f[2] = a.z; f[3] = a.w;
  f[4] = b.x; f[5] = b.y; f[6] = b.z; f[7] = b.w;
}

// Tile geometry.  A warp is 8 token groups (ty) x 4 expert groups (tx);
// thread (ty, tx) owns TM consecutive tokens and TN experts taken as TN/4
// float4 groups spaced 16 experts apart, so each operand read of a warp is
// one contiguous, conflict-free shared-memory wavefront.  WT x WE warps per
// CTA: BT = 8 TM WT tokens x BE = 4 TN WE experts.
template <typename Tin, int TM, int TN, int WT, int WE>
struct LogitsCfg {
  static constexpr int BT = 8 * TM * WT;
  static constexpr int BE = 4 * TN * WE;
  static constexpr int kRows = BT + BE;
  static constexpr int kThreads = 32 * WT * WE;
  static constexpr int kRowBytes = kKc * static_cast<int>(sizeof(Tin)) + 16;
  static constexpr int kVecs = kKc * static_cast<int>(sizeof(Tin)) / 16;
  static constexpr int kElemsPerVec = 16 / static_cast<int>(sizeof(Tin));
  static constexpr int kRawStage = kRows * kRowBytes;
  static constexpr int kCbuf = kKc * kRows;  // floats in one widened chunk
  static constexpr int kSmem = kStagesL * kRawStage + 2 * kCbuf * 4;
};

// Each score is one fma chain over k = 0 .. d-1 in order.  Raw chunks of 32 k
// stream through a cp.async ring; each chunk is widened once into a k-major
// fp32 buffer buf[k][row] (rows: BT tokens, then BE experts) and every thread
// then reads TM + TN operands per k for TM x TN fmas.
template <typename Tin, int TM, int TN, int WT, int WE>
__global__ void __launch_bounds__(LogitsCfg<Tin, TM, TN, WT, WE>::kThreads)
    logits_kernel(const Tin* __restrict__ h, const Tin* __restrict__ w, int T,
                  int d, int E, float* __restrict__ z, uint32_t* __restrict__ zw, int nz) {
  using C = LogitsCfg<Tin, TM, TN, WT, WE>;
  constexpr int BT = C::BT, BE = C::BE, R = C::kRows, NT = C::kThreads;
  extern __shared__ __align__(16) uint8_t smem_l[];
  grid_dep_wait();
  grid_dep_launch();
  if (zw != nullptr && blockIdx.x == 0 && blockIdx.y == 0)
    for (int i = threadIdx.x; i < nz; i += blockDim.x) zw[i] = 0u;
  float* cbuf = reinterpret_cast<float*>(smem_l + kStagesL * C::kRawStage);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int ty = lane >> 2, tx = lane & 3;
  const int wt = warp / WE, we = warp % WE;
  const int my_t = wt * (8 * TM) + ty * TM;  // first token row of this thread
  const int my_e = we * (4 * TN) + 4 * tx;   // first expert row of group 0
  const int t0 = blockIdx.x * BT;
  const int e0 = blockIdx.y * BE;
  const int nchunks = d / kKc;

  auto issue = [&](int c) {
    uint8_t* st = smem_l + (c % kStagesL) * C::kRawStage;
    const int k0 = c * kKc;
    for (int v = threadIdx.x; v < R * C::kVecs; v += NT) {
      const int r = v / C::kVecs, q = v % C::kVecs;
      const bool is_h = r < BT;
      const int idx = is_h ? t0 + r : e0 + (r - BT);
      const bool ok = idx < (is_h ? T : E);
      const Tin* base = is_h ? h : w;
      cp_async16(st + r * C::kRowBytes + q * 16,
                 base + (ok ? static_cast<int64_t>(idx) * d + k0 + q * C::kElemsPerVec : 0),
                 ok);
    }
  };
  auto widen = [&](int c, float* buf) {
    const uint8_t* st = smem_l + (c % kStagesL) * C::kRawStage;
    for (int v = threadIdx.x; v < R * (kKc / 8); v += NT) {
      const int r = v % R, q = v / R;  // consecutive rows per warp
      float f[8];
      widen8(st + r * C::kRowBytes + q * 8 * sizeof(Tin), f, static_cast<const Tin*>(nullptr));
#pragma unroll
      for (int i = 0; i < 8; ++i) buf[(q * 8 + i) * R + r] = f[i];
    }
  };

  float acc[TM][TN];
#pragma unroll
  for (int i = 0; i < TM; ++i)
#pragma unroll
    for (int j = 0; j < TN; ++j) acc[i][j] = 0.f;

#pragma unroll
  for (int c = 0; c < kStagesL - 1; ++c) {
    if (c < nchunks) issue(c);
    cp_async_commit();
  }
  for (int c = 0; c < nchunks; ++c) {
    cp_async_wait<kStagesL - 2>();
    __syncthreads();  // raw chunk c visible; iteration c-1 finished everywhere
    if (c + kStagesL - 1 < nchunks) issue(c + kStagesL - 1);
    cp_async_commit();
    float* buf = cbuf + (c & 1) * C::kCbuf;
    widen(c, buf);
    __syncthreads();
#pragma unroll 8
    for (int kk = 0; kk < kKc; ++kk) {
      const float* row = buf + kk * R;
      float hv[TM], wv[TN];
      if constexpr (TM == 4) {
        const float4 q4 = *reinterpret_cast<const float4*>(row + my_t);
        hv[0] = q4.x; hv[1] = q4.y; hv[2] = q4.z; hv[3] = q4.w;
      } else {
#pragma unroll
        for (int i = 0; i < TM; ++i) hv[i] = row[my_t + i];
      }
#pragma unroll
      for (int g = 0; g < TN / 4; ++g) {
        const float4 q4 = *reinterpret_cast<const float4*>(row + BT + my_e + 16 * g);
        wv[4 * g] = q4.x; wv[4 * g + 1] = q4.y; wv[4 * g + 2] = q4.z; wv[4 * g + 3] = q4.w;
      }
#pragma unroll
      for (int i = 0; i < TM; ++i)
#pragma unroll
        for (int j = 0; j < TN; ++j) acc[i][j] = __fmaf_rn(hv[i], wv[j], acc[i][j]);
    }
  }
  cp_async_wait<0>();
#pragma unroll
  for (int i = 0; i < TM; ++i) {
    const int t = t0 + my_t + i;
    if (t >= T) continue;
#pragma unroll
    for (int j = 0; j < TN; ++j) {
      const int e = e0 + my_e + 16 * (j / 4) + (j % 4);
      if (e < E) z[static_cast<int64_t>(t) * E + e] = acc[i][j];
    }
  }
}

template <typename Tin, int TM, int TN, int WT, int WE>
cudaError_t launch_logits_tile(const Tin* h, const Tin* w, int T, int d, int E,
                               float* z, uint32_t* zw, int nz, cudaStream_t s) {
  using C = LogitsCfg<Tin, TM, TN, WT, WE>;
  auto kern = logits_kernel<Tin, TM, TN, WT, WE>;
  if (C::kSmem > 48 * 1024) {
    const cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmem);
    if (e != cudaSuccess) return e;
  }
  const dim3 g((T + C::BT - 1) / C::BT, (E + C::BE - 1) / C::BE);
  kern<<<g, C::kThreads, C::kSmem, s>>>(h, w, T, d, E, z, zw, nz);
  return cudaGetLastError();
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
  grid_dep_wait();
  grid_dep_launch();
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

// Selection whose counts come from the router scores (the threshold-based
// count rules, App. B): one warp per token derives k_t from the routing mass
// softmax(z_t) in the fp32 order include/reflex.h states (exp_cw, lane sums
// in ascending expert order, xor-butterfly over the lanes), writes it to
// kout (and adds it to ksum), then selects TopK(z_t, k_t) and the weights as
// select_kernel does.  rule 1 = Top-p (smallest prefix of ranks whose mass
// reaches thr), rule 2 = expert threshold (experts whose mass exceeds thr);
// either clipped to [k_lo, min(k_hi, E)].  ids == nullptr: counts only.
template <int NPL>
__global__ void __launch_bounds__(kSelWarps * 32)
    select_rule_kernel(const float* __restrict__ z, int T, int E, int k_hi, int k_lo,
                       int rule, float thr, int k_max, int renorm,
                       int32_t* __restrict__ kout, unsigned long long* __restrict__ ksum,
                       int32_t* __restrict__ ids, float* __restrict__ alpha) {
  __shared__ float s_z[kSelWarps][32];
  __shared__ int32_t s_e[kSelWarps][32];
  grid_dep_wait();
  grid_dep_launch();
  const int wid = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t = blockIdx.x * kSelWarps + wid;
  if (t >= T) return;
  const int kcap = k_hi < E ? k_hi : E;
  const int klo = k_lo < kcap ? k_lo : kcap;
  float zv[NPL];
  unsigned long long key[NPL];
  const float* zt = z + static_cast<int64_t>(t) * E;
  float m = -INFINITY;
#pragma unroll
  for (int i = 0; i < NPL; ++i) {
    const int e = lane + 32 * i;
    if (e < E) {
      float v = zt[e];
      v = (v == 0.0f) ? 0.0f : v;
      zv[i] = v;
      key[i] = (static_cast<unsigned long long>(order_bits(v)) << 32) |
               static_cast<unsigned long long>(0xffffffffu - static_cast<uint32_t>(e));
      m = fmaxf(m, v);
    } else {
      zv[i] = -INFINITY;
      key[i] = 0ull;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
  // u_e = exp(z_e - m); S = lane sums in ascending expert order, then the
  // xor-butterfly (every lane ends with the same bits)
  float u[NPL];
  float S = 0.0f;
#pragma unroll
  for (int i = 0; i < NPL; ++i) {
    u[i] = (lane + 32 * i < E) ? exp_cw(__fsub_rn(zv[i], m)) : 0.0f;
    S = __fadd_rn(S, u[i]);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) S = __fadd_rn(S, __shfl_xor_sync(0xffffffffu, S, o));
  int kt = kcap;
  if (rule == 2) {
    int cnt = 0;
#pragma unroll
    for (int i = 0; i < NPL; ++i)
      cnt += __popc(__ballot_sync(0xffffffffu,
                                  lane + 32 * i < E && __fdiv_rn(u[i], S) > thr));
    kt = cnt < klo ? klo : (cnt > kcap ? kcap : cnt);
  }
  float c = 0.0f;  // Top-p: mass of the ranks taken so far
  // the ranks are needed to select, and by Top-p to count
  const int rounds = (ids != nullptr || rule == 1) ? kt : 0;
  for (int j = 0; j < rounds && j < kt; ++j) {
    unsigned long long best = key[0];
#pragma unroll
    for (int i = 1; i < NPL; ++i) best = key[i] > best ? key[i] : best;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const unsigned long long other = __shfl_xor_sync(0xffffffffu, best, o);
      best = other > best ? other : best;
    }
    const int e = static_cast<int>(0xffffffffu - static_cast<uint32_t>(best & 0xffffffffull));
    const float ze = from_order_bits(static_cast<uint32_t>(best >> 32));
    if ((e & 31) == lane) {
#pragma unroll
      for (int i = 0; i < NPL; ++i)
        if (i == (e >> 5)) key[i] = 0ull;
    }
    if (lane == 0) {
      s_e[wid][j] = e;
      s_z[wid][j] = ze;
    }
    if (rule == 1) {
      c = __fadd_rn(c, exp_cw(__fsub_rn(ze, m)));
      if (j + 1 >= klo && __fdiv_rn(c, S) >= thr) kt = j + 1;  // ends the loop
    }
  }
  if (lane == 0) {
    kout[t] = kt;
    if (ksum != nullptr) atomicAdd(ksum, static_cast<unsigned long long>(kt));
  }
  if (ids == nullptr) return;
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

// Short-batch variant: too few (token, expert) chains to fill the GPU with
// the widened-buffer tiles, so each CTA (4 warps) keeps 8 TM tokens x 64
// experts, one 4-stage ring of 32-k raw chunks, and widens operands at use
// (no extra pass, one barrier per chunk).  Thread (warp w, lane l) owns
// tokens t0 + (l >> 2) + 8 i and experts e0 + 16 w + (l & 3) + 4 j; with
// rows padded by 16 bytes each 16-byte operand read of a warp is
// conflict-free.
constexpr int kStagesS = 4;
constexpr int kThreadsS = 128;

template <typename Tin>
__device__ __forceinline__ void row8(const uint8_t* p, float* f) {
  widen8(p, f, static_cast<const Tin*>(nullptr));
}

template <typename Tin, int TM>
__global__ void __launch_bounds__(kThreadsS)
    logits_short_kernel(const Tin* __restrict__ h, const Tin* __restrict__ w,
                        int T, int d, int E, float* __restrict__ z,
                        uint32_t* __restrict__ zw, int nz) {
  constexpr int BT = 8 * TM, BE = 64;
  constexpr int kRowBytes = kKc * static_cast<int>(sizeof(Tin)) + 16;
  constexpr int kVecs = kKc * static_cast<int>(sizeof(Tin)) / 16;
  constexpr int kElemsPerVec = 16 / static_cast<int>(sizeof(Tin));
  constexpr int kHBytes = BT * kRowBytes;
  constexpr int kStageBytes = (BT + BE) * kRowBytes;
  extern __shared__ __align__(16) uint8_t smem_s[];
  grid_dep_wait();
  grid_dep_launch();
  if (zw != nullptr && blockIdx.x == 0 && blockIdx.y == 0)
    for (int i = threadIdx.x; i < nz; i += blockDim.x) zw[i] = 0u;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int ty = lane >> 2, tx = lane & 3;
  const int t0 = blockIdx.x * BT;
  const int e0 = blockIdx.y * BE;
  const int nchunks = d / kKc;

  auto issue = [&](int c) {
    uint8_t* st = smem_s + (c % kStagesS) * kStageBytes;
    const int k0 = c * kKc;
    for (int v = threadIdx.x; v < (BT + BE) * kVecs; v += kThreadsS) {
      const int r = v / kVecs, q = v % kVecs;
      const bool is_h = r < BT;
      const int idx = is_h ? t0 + r : e0 + (r - BT);
      const bool ok = idx < (is_h ? T : E);
      const Tin* base = is_h ? h : w;
      cp_async16(st + r * kRowBytes + q * 16,
                 base + (ok ? static_cast<int64_t>(idx) * d + k0 + q * kElemsPerVec : 0), ok);
    }
  };

  float acc[TM][4];
#pragma unroll
  for (int i = 0; i < TM; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

#pragma unroll
  for (int c = 0; c < kStagesS - 1; ++c) {
    if (c < nchunks) issue(c);
    cp_async_commit();
  }
  for (int c = 0; c < nchunks; ++c) {
    cp_async_wait<kStagesS - 2>();
    __syncthreads();
    if (c + kStagesS - 1 < nchunks) issue(c + kStagesS - 1);
    cp_async_commit();
    const uint8_t* st = smem_s + (c % kStagesS) * kStageBytes;
#pragma unroll
    for (int kv = 0; kv < kKc / 8; ++kv) {
      float hv[TM][8], wv[4][8];
#pragma unroll
      for (int i = 0; i < TM; ++i)
        row8<Tin>(st + (ty + 8 * i) * kRowBytes + kv * 8 * sizeof(Tin), hv[i]);
#pragma unroll
      for (int j = 0; j < 4; ++j)
        row8<Tin>(st + kHBytes + (16 * warp + tx + 4 * j) * kRowBytes + kv * 8 * sizeof(Tin),
                  wv[j]);
#pragma unroll
      for (int kk = 0; kk < 8; ++kk)
#pragma unroll
        for (int i = 0; i < TM; ++i)
#pragma unroll
          for (int j = 0; j < 4; ++j)
            acc[i][j] = __fmaf_rn(hv[i][kk], wv[j][kk], acc[i][j]);
    }
  }
  cp_async_wait<0>();
#pragma unroll
  for (int i = 0; i < TM; ++i) {
    const int t = t0 + ty + 8 * i;
    if (t >= T) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int e = e0 + 16 * warp + tx + 4 * j;
      if (e < E) z[static_cast<int64_t>(t) * E + e] = acc[i][j];
    }
  }
}

template <typename Tin, int TM>
cudaError_t launch_logits_short(const Tin* h, const Tin* w, int T, int d, int E,
                                float* z, uint32_t* zw, int nz, cudaStream_t s) {
  constexpr int kRowBytes = kKc * static_cast<int>(sizeof(Tin)) + 16;
  constexpr int smem = kStagesS * (8 * TM + 64) * kRowBytes;
  auto kern = logits_short_kernel<Tin, TM>;
  if (smem > 48 * 1024) {
    const cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
  }
  const dim3 g((T + 8 * TM - 1) / (8 * TM), (E + 63) / 64);
  kern<<<g, kThreadsS, smem, s>>>(h, w, T, d, E, z, zw, nz);
  return cudaGetLastError();
}

// ---- bf16 scores with mixed-precision fma ----------------------------------
// fma.rn.f32.bf16 d, a, b, c rounds a*b + c once to fp32 with bf16 a, b and
// fp32 c, d.  A bf16 x bf16 product is exact in fp32, so every step equals
// fma(widen(a), widen(b), c) bit for bit and the chain needs no widening
// instructions: operands go from shared memory straight into the fma.
__device__ __forceinline__ void fma_lo(float& acc, uint32_t a2, uint32_t b2) {
  asm("{\n\t.reg .b16 al, ah, bl, bh;\n\t"
      "mov.b32 {al, ah}, %1;\n\t"
      "mov.b32 {bl, bh}, %2;\n\t"
      "fma.rn.f32.bf16 %0, al, bl, %0;\n\t}"
      : "+f"(acc)
      : "r"(a2), "r"(b2));
}
__device__ __forceinline__ void fma_hi(float& acc, uint32_t a2, uint32_t b2) {
  asm("{\n\t.reg .b16 al, ah, bl, bh;\n\t"
      "mov.b32 {al, ah}, %1;\n\t"
      "mov.b32 {bl, bh}, %2;\n\t"
      "fma.rn.f32.bf16 %0, ah, bh, %0;\n\t}"
      : "+f"(acc)
      : "r"(a2), "r"(b2));
}

// Tile geometry.  A warp is LY token lanes x LX expert lanes (LY LX = 32);
// lane (ty, tx) owns tokens ty + LY i (i < TM) and experts tx + LX j
// (j < TN) of the warp tile, so for fixed (i, j) the warp reads LY (resp.
// LX) consecutive rows; with rows padded to 80 bytes any 8 consecutive rows
// start in distinct 16-byte bank groups and each 16-byte operand read is one
// shared-memory wavefront.  WT x WE warps per CTA.
template <int LY, int TM, int TN, int WT, int WE, int S, int KC>
struct MxCfg {
  static constexpr int LX = 32 / LY;
  static constexpr int BT = LY * TM * WT;   // tokens per CTA
  static constexpr int BE = LX * TN * WE;   // experts per CTA
  static constexpr int NT = 32 * WT * WE;
  static constexpr int kRowBytes = KC * 2 + 16;
  static constexpr int kStage = (BT + BE) * kRowBytes;
  static constexpr int kSmem = S * kStage;
};

// Each thread keeps TM x TN chains; per 8-k step it reads TM token and TN
// expert vectors of 8 bf16 and issues 8 TM TN fmas, every chain advancing
// over k = 0 .. d-1 in order (within a 32-bit word: even k, then odd k).
// Raw KC-k chunks stream through an S-stage cp.async ring.
template <int LY, int TM, int TN, int WT, int WE, int S, int KC>
__global__ void __launch_bounds__(MxCfg<LY, TM, TN, WT, WE, S, KC>::NT)
    logits_mx_kernel(const __nv_bfloat16* __restrict__ h,
                     const __nv_bfloat16* __restrict__ w, int T, int d, int E,
                     float* __restrict__ z, uint32_t* __restrict__ zw, int nz) {
  using C = MxCfg<LY, TM, TN, WT, WE, S, KC>;
  constexpr int LX = C::LX, BT = C::BT, BE = C::BE, NT = C::NT;
  constexpr int kRB = C::kRowBytes;
  constexpr int kVecs = KC / 8;  // 16-byte vectors per row per chunk
  extern __shared__ __align__(16) uint8_t smem_m[];
  grid_dep_wait();
  grid_dep_launch();
  if (zw != nullptr && blockIdx.x == 0 && blockIdx.y == 0)
    for (int i = threadIdx.x; i < nz; i += blockDim.x) zw[i] = 0u;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int ty = lane / LX, tx = lane % LX;
  const int wt = warp / WE, we = warp % WE;
  const int rt = wt * (LY * TM) + ty;       // first token row of this thread
  const int re = we * (LX * TN) + tx;       // first expert row
  const int t0 = blockIdx.x * BT;
  const int e0 = blockIdx.y * BE;
  const int nchunks = d / KC;

  auto issue = [&](int c) {
    uint8_t* st = smem_m + (c % S) * C::kStage;
    const int k0 = c * KC;
    for (int v = threadIdx.x; v < (BT + BE) * kVecs; v += NT) {
      const int r = v / kVecs, q = v % kVecs;
      const bool is_h = r < BT;
      const int idx = is_h ? t0 + r : e0 + (r - BT);
      const bool ok = idx < (is_h ? T : E);
      const __nv_bfloat16* base = is_h ? h : w;
      cp_async16(st + r * kRB + q * 16,
                 base + (ok ? static_cast<int64_t>(idx) * d + k0 + q * 8 : 0), ok);
    }
  };

  float acc[TM][TN];
#pragma unroll
  for (int i = 0; i < TM; ++i)
#pragma unroll
    for (int j = 0; j < TN; ++j) acc[i][j] = 0.f;

#pragma unroll
  for (int c = 0; c < S - 1; ++c) {
    if (c < nchunks) issue(c);
    cp_async_commit();
  }
  for (int c = 0; c < nchunks; ++c) {
    cp_async_wait<S - 2>();
    __syncthreads();  // chunk c visible; chunk c-1's slot free everywhere
    if (c + S - 1 < nchunks) issue(c + S - 1);
    cp_async_commit();
    const uint8_t* st = smem_m + (c % S) * C::kStage;
    const uint8_t* hrow = st + rt * kRB;
    const uint8_t* wrow = st + (BT + re) * kRB;
#pragma unroll
    for (int kv = 0; kv < kVecs; ++kv) {
      uint4 hv[TM], wv[TN];
#pragma unroll
      for (int i = 0; i < TM; ++i)
        hv[i] = *reinterpret_cast<const uint4*>(hrow + (LY * i) * kRB + kv * 16);
#pragma unroll
      for (int j = 0; j < TN; ++j)
        wv[j] = *reinterpret_cast<const uint4*>(wrow + (LX * j) * kRB + kv * 16);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
#pragma unroll
        for (int i = 0; i < TM; ++i) {
          const uint32_t a2 = q == 0 ? hv[i].x : q == 1 ? hv[i].y : q == 2 ? hv[i].z : hv[i].w;
#pragma unroll
          for (int j = 0; j < TN; ++j) {
            const uint32_t b2 = q == 0 ? wv[j].x : q == 1 ? wv[j].y : q == 2 ? wv[j].z : wv[j].w;
            fma_lo(acc[i][j], a2, b2);
          }
        }
#pragma unroll
        for (int i = 0; i < TM; ++i) {
          const uint32_t a2 = q == 0 ? hv[i].x : q == 1 ? hv[i].y : q == 2 ? hv[i].z : hv[i].w;
#pragma unroll
          for (int j = 0; j < TN; ++j) {
            const uint32_t b2 = q == 0 ? wv[j].x : q == 1 ? wv[j].y : q == 2 ? wv[j].z : wv[j].w;
            fma_hi(acc[i][j], a2, b2);
          }
        }
      }
    }
  }
  cp_async_wait<0>();
#pragma unroll
  for (int i = 0; i < TM; ++i) {
    const int t = t0 + rt + LY * i;
    if (t >= T) continue;
#pragma unroll
    for (int j = 0; j < TN; ++j) {
      const int e = e0 + re + LX * j;
      if (e < E) z[static_cast<int64_t>(t) * E + e] = acc[i][j];
    }
  }
}

// ---- bf16 scores, whole rows resident --------------------------------------
// Few chains per SM: the ring kernel above syncs its CTA once per 32-k chunk
// while each thread advances only one or two chains, so barriers and refill
// latency dominate and a chain step costs several times the fma latency.
// Here a CTA keeps all d columns of its BT token rows and BE expert rows in
// shared memory (rows padded by 16 bytes, so any 8 consecutive rows start in
// distinct 16-byte bank groups).  Every thread issues its share of all row
// chunks up front with cp.async, chunk by chunk, and hands each chunk to that
// chunk's mbarrier (cp.async.mbarrier.arrive.noinc): a chunk's phase completes
// once every thread's copies into it have landed.  The threads then walk the
// chunks in order, waiting only for the chunk they read next, with the
// operands of step s + 1 loaded while step s runs its fmas: no slot reuse, no
// block-wide barrier in the k loop, and one chain step costs about one fma
// latency.  Same thread geometry and fma order as the ring kernel, so the
// scores are the same bits.  (One 512-byte bulk copy per row chunk measured
// about 50 ns per copy on GB300, three times slower than the cp.async path.)
constexpr int kResChunkK = 256;   // k per chunk; d must be a multiple
constexpr int kResSteps = kResChunkK / 8;  // 16-byte steps per row per chunk
constexpr int kResMaxChunks = 16;
constexpr int kResBarBytes = 128;
constexpr uint64_t kL2PrefetchPiece = 64u * 1024u;
constexpr uint64_t kResWaitNs = 2000000000ull;
constexpr uint64_t kResDrainNs = 1000000000ull;

template <int LY, int TM, int TN, int WT, int WE>
struct ResCfg {
  static constexpr int LX = 32 / LY;
  static constexpr int BT = LY * TM * WT;  // tokens per CTA
  static constexpr int BE = LX * TN * WE;  // experts per CTA
  static constexpr int NT = 32 * WT * WE;
  static constexpr int kRows = BT + BE;
  static size_t smem(int d) {
    return kResBarBytes + static_cast<size_t>(kRows) * (2 * static_cast<size_t>(d) + 16);
  }
};

__device__ __forceinline__ void cp_async_arrive_noinc(uint32_t bar) {
  asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];" ::"r"(bar) : "memory");
}

template <int TM, int TN>
struct MxOps {
  uint4 h[TM], w[TN];
};
template <int TM, int TN>
__device__ __forceinline__ void mx_load(MxOps<TM, TN>& o, const uint8_t* hrow,
                                        const uint8_t* wrow, int hstride, int wstride, int off) {
#pragma unroll
  for (int i = 0; i < TM; ++i) o.h[i] = *reinterpret_cast<const uint4*>(hrow + i * hstride + off);
#pragma unroll
  for (int j = 0; j < TN; ++j) o.w[j] = *reinterpret_cast<const uint4*>(wrow + j * wstride + off);
}
// 8 k of every chain: even k then odd k of each 32-bit word, words in order
template <int TM, int TN>
__device__ __forceinline__ void mx_fma8(float (&acc)[TM][TN], const MxOps<TM, TN>& o) {
#pragma unroll
  for (int q = 0; q < 4; ++q) {
#pragma unroll
    for (int i = 0; i < TM; ++i) {
      const uint32_t a2 = q == 0 ? o.h[i].x : q == 1 ? o.h[i].y : q == 2 ? o.h[i].z : o.h[i].w;
#pragma unroll
      for (int j = 0; j < TN; ++j) {
        const uint32_t b2 = q == 0 ? o.w[j].x : q == 1 ? o.w[j].y : q == 2 ? o.w[j].z : o.w[j].w;
        fma_lo(acc[i][j], a2, b2);
      }
    }
#pragma unroll
    for (int i = 0; i < TM; ++i) {
      const uint32_t a2 = q == 0 ? o.h[i].x : q == 1 ? o.h[i].y : q == 2 ? o.h[i].z : o.h[i].w;
#pragma unroll
      for (int j = 0; j < TN; ++j) {
        const uint32_t b2 = q == 0 ? o.w[j].x : q == 1 ? o.w[j].y : q == 2 ? o.w[j].z : o.w[j].w;
        fma_hi(acc[i][j], a2, b2);
      }
    }
  }
}

// Each CTA hands its share of [pf.base, pf.base + pf.bytes) to the L2 as
// bulk prefetches (the TMA unit moves them; no thread waits for them).
__device__ __forceinline__ void l2_prefetch_share(const L2Prefetch& pf) {
  if (pf.bytes == 0) return;
  const uint64_t nct = static_cast<uint64_t>(gridDim.x) * gridDim.y;
  const uint64_t cid = static_cast<uint64_t>(blockIdx.y) * gridDim.x + blockIdx.x;
  uint64_t chunk = (pf.bytes + nct - 1) / nct;
  chunk = (chunk + 4095u) & ~static_cast<uint64_t>(4095u);
  const uint64_t b0 = cid * chunk;
  const uint64_t b1 = b0 + chunk < pf.bytes ? b0 + chunk : pf.bytes;
  const uint8_t* base = static_cast<const uint8_t*>(pf.base);
  for (uint64_t b = b0; b < b1; b += kL2PrefetchPiece) {
    const uint32_t n = static_cast<uint32_t>(b1 - b < kL2PrefetchPiece ? b1 - b : kL2PrefetchPiece);
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(base + b), "r"(n)
                 : "memory");
  }
}

template <int LY, int TM, int TN, int WT, int WE>
__global__ void __launch_bounds__(ResCfg<LY, TM, TN, WT, WE>::NT, 1)
    logits_res_kernel(const __nv_bfloat16* __restrict__ h,
                      const __nv_bfloat16* __restrict__ w, int T, int d, int E,
                      float* __restrict__ z, uint32_t* __restrict__ zw, int nz,
                      uint32_t* __restrict__ err, L2Prefetch pf) {
  using C = ResCfg<LY, TM, TN, WT, WE>;
  constexpr int LX = C::LX, BT = C::BT, BE = C::BE, NT = C::NT;
  constexpr int kVecs = C::kRows * kResSteps;  // 16-byte copies per chunk
  extern __shared__ __align__(128) uint8_t smem_r[];
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem_r);
  uint8_t* rows = smem_r + kResBarBytes;
  grid_dep_wait();
  grid_dep_launch();
  // CTA (0, 0) clears the header words when it starts; a wait of another
  // CTA can only expire (and set an error bit) kResWaitNs after that CTA
  // started, and the grid is at most two waves of CTAs that start within
  // microseconds of each other, so the clear comes first.  Callers that need
  // the order guaranteed clear the word in stream order and pass nz = 0.
  if (zw != nullptr && blockIdx.x == 0 && blockIdx.y == 0)
    for (int i = threadIdx.x; i < nz; i += blockDim.x) zw[i] = 0u;
  const int pitch = 2 * d + 16;
  const int nch = d / kResChunkK;  // 1 .. kResMaxChunks (host check)
  const int t0 = blockIdx.x * BT, e0 = blockIdx.y * BE;
  const int nt = min(BT, T - t0), ne = min(BE, E - e0);
  if (threadIdx.x == 0) {
    for (int c = 0; c < nch; ++c) mbar_init(&bars[c], NT);
    fence_mbar_init();
  }
  __syncthreads();
  for (int c = 0; c < nch; ++c) {
    const int k0 = c * kResChunkK;
    for (int v = threadIdx.x; v < kVecs; v += NT) {
      const int r = v / kResSteps, q = v % kResSteps;
      const bool is_h = r < BT;
      const int idx = is_h ? r : r - BT;
      const bool ok = idx < (is_h ? nt : ne);  // rows past T or E: zero fill
      const __nv_bfloat16* src =
          ok ? (is_h ? h + static_cast<int64_t>(t0 + idx) * d
                     : w + static_cast<int64_t>(e0 + idx) * d) + k0 + 8 * q
             : h;
      cp_async16(rows + r * pitch + 2 * k0 + 16 * q, src, ok);
    }
    cp_async_arrive_noinc(smem_addr(&bars[c]));
  }
  if (threadIdx.x == 0) l2_prefetch_share(pf);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int ty = lane / LX, tx = lane % LX;
  const int wt = warp / WE, we = warp % WE;
  const int rt = wt * (LY * TM) + ty;  // first token row of this thread
  const int re = we * (LX * TN) + tx;  // first expert row
  const uint8_t* hrow = rows + rt * pitch;
  const uint8_t* wrow = rows + (BT + re) * pitch;
  float acc[TM][TN];
#pragma unroll
  for (int i = 0; i < TM; ++i)
#pragma unroll
    for (int j = 0; j < TN; ++j) acc[i][j] = 0.f;
  bool ok = mbar_wait(&bars[0], 0u, nullptr, kResWaitNs);
  MxOps<TM, TN> ops[2];
  if (ok) mx_load(ops[0], hrow, wrow, LY * pitch, LX * pitch, 0);
  for (int c = 0; c < nch && ok; ++c) {
    const int off = 2 * c * kResChunkK;
#pragma unroll
    for (int s = 0; s < kResSteps; ++s) {
      if (s + 1 < kResSteps) {
        mx_load(ops[(s + 1) & 1], hrow, wrow, LY * pitch, LX * pitch, off + 16 * (s + 1));
      } else if (c + 1 < nch) {
        ok = mbar_wait(&bars[c + 1], 0u, nullptr, kResWaitNs);
        if (ok) mx_load(ops[(s + 1) & 1], hrow, wrow, LY * pitch, LX * pitch, off + 16 * (s + 1));
      }
      mx_fma8<TM, TN>(acc, ops[s & 1]);
    }
  }
  if (!ok) {
    // every copy into this CTA's shared memory must land before it exits;
    // the thread's scores are incomplete and are stored as -inf (never left
    // as whatever an earlier call wrote there)
    set_err(err, kErrTimeout);
    for (int c = 0; c < nch; ++c) mbar_wait(&bars[c], 0u, nullptr, kResDrainNs);
  }
#pragma unroll
  for (int i = 0; i < TM; ++i) {
    const int t = t0 + rt + LY * i;
    if (t >= T) continue;
#pragma unroll
    for (int j = 0; j < TN; ++j) {
      const int e = e0 + re + LX * j;
      if (e < E) z[static_cast<int64_t>(t) * E + e] = ok ? acc[i][j] : -INFINITY;
    }
  }
}

template <int LY, int TM, int TN, int WT, int WE>
cudaError_t launch_logits_res(const __nv_bfloat16* h, const __nv_bfloat16* w, int T, int d,
                              int E, float* z, uint32_t* zw, int nz, uint32_t* err,
                              const L2Prefetch& pf, cudaStream_t s) {
  using C = ResCfg<LY, TM, TN, WT, WE>;
  if (d % kResChunkK != 0 || d / kResChunkK > kResMaxChunks) return cudaErrorInvalidValue;
  auto kern = logits_res_kernel<LY, TM, TN, WT, WE>;
  const size_t smem = C::smem(d);
  const cudaError_t e =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const dim3 g((T + C::BT - 1) / C::BT, (E + C::BE - 1) / C::BE);
  kern<<<g, C::NT, smem, s>>>(h, w, T, d, E, z, zw, nz, err, pf);
  return cudaGetLastError();
}

// ---- screened selection (bf16 inputs, weights renormalised over the set) --
// The tensor cores give every score z~[t, e] (fp32 accumulators, split-K
// partial sums added in slice order).  Both z~ and the canonical chain z lie
// within their error bounds of the exact dot product: for the chain (one
// rounding per fma, d steps) |z - z*| <= gamma_d sum_k |h_k w_k| with
// gamma_d = d u / (1 - d u), u = 2^-24; the tensor-core estimate is taken to
// err by at most 2^-12 sum |h_k w_k| (about 4x a crude worst case of a few
// units in the last place per 16-product step, and far above what is
// observed), plus one rounding per split-K slice.  With sum |h_k w_k| <=
// ||h_t|| ||w_e|| (Cauchy-Schwarz) every z lies in [lo_e, hi_e] = z~_e -/+
// delta_e.  Let L be the k_t-th largest lo: at least k_t experts have z >= L,
// so an expert with hi_e < L cannot be among the k_t largest; the candidates
// C = {e : hi_e >= L} contain the canonical TopK set.  Their scores are
// recomputed with the canonical chain (the same fma.rn.f32.bf16 sequence as
// the score kernels), and the TopK over C (same keys, same tie rule) is the
// TopK over all experts.  Scores of the other experts stay tensor-core
// estimates in z.  One warp per token; a token with more than 32 candidates
// recomputes every expert.
constexpr int kScreenWarps = 8;

// ||w_e||_2, rounded up (every step of the fp32 sum of squares is covered by
// the factors below).
// The first kernel of a screened forward: it also clears zero_words[0, nz).
__global__ void __launch_bounds__(256)
    wnorm_kernel(const __nv_bfloat16* __restrict__ w, int E, int d, float* __restrict__ nw,
                 uint32_t* __restrict__ zw, int nz) {
  grid_dep_wait();
  grid_dep_launch();
  if (zw != nullptr && blockIdx.x == 0)
    for (int i = threadIdx.x; i < nz; i += blockDim.x) zw[i] = 0u;
  const int lane = threadIdx.x & 31;
  const int e = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (e >= E) return;
  const uint4* row = reinterpret_cast<const uint4*>(w + static_cast<int64_t>(e) * d);
  float ss = 0.f;
  for (int v = lane; v < d / 8; v += 32) {
    const uint4 q = row[v];
    const uint32_t wd[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float a = __uint_as_float(wd[i] << 16), b = __uint_as_float(wd[i] & 0xffff0000u);
      ss = fmaf(a, a, ss);
      ss = fmaf(b, b, ss);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  if (lane == 0) nw[e] = sqrtf(ss * (1.0f + 0x1p-10f)) * (1.0f + 0x1p-20f);
}

// canonical chain of one (token, expert) pair: fma over k = 0 .. d-1 in
// order.  The token row comes from shared memory (the same address in every
// lane), the expert row from L2.  (A ring keeping 8-16 expert-row loads in
// flight per lane made short batches faster but cost occupancy at 8192 and
// more tokens, where the screen is used.)
constexpr int kScreenDMultiple = 128;  // d of the screened path (as tested)
__device__ __forceinline__ float chain_bf16(const uint4* __restrict__ hs,
                                            const __nv_bfloat16* __restrict__ we, int d) {
  const uint4* wv = reinterpret_cast<const uint4*>(we);
  const int nv = d / 8;
  float acc = 0.f;
#pragma unroll 4
  for (int v = 0; v < nv; ++v) {
    const uint4 a = hs[v], b = __ldg(wv + v);
    fma_lo(acc, a.x, b.x);
    fma_hi(acc, a.x, b.x);
    fma_lo(acc, a.y, b.y);
    fma_hi(acc, a.y, b.y);
    fma_lo(acc, a.z, b.z);
    fma_hi(acc, a.z, b.z);
    fma_lo(acc, a.w, b.w);
    fma_hi(acc, a.w, b.w);
  }
  return acc;
}

// The same chain with 32-byte expert-row loads (two in flight per lane):
// half the load instructions and L1 requests of the 16-byte form, whose
// warp loads each touch a different row per lane (LLaDA2.0-mini routing
// 113.6 -> 107.6 us).  Needs the row 32-byte aligned and d % 32 == 0 (the
// loop takes the 32-byte steps in pairs; the screened path has d % 128 == 0).
__device__ __forceinline__ float chain_bf16_wide(const uint4* __restrict__ hs,
                                                 const __nv_bfloat16* __restrict__ we, int d) {
  const uint32_t* wp = reinterpret_cast<const uint32_t*>(we);
  const int n = d / 16;  // 32-byte steps (d % 32 == 0 keeps the pair whole)
  float acc = 0.f;
  for (int v0 = 0; v0 < n; v0 += 2) {
    uint32_t b[2][8];
#pragma unroll
    for (int u = 0; u < 2; ++u)
      asm("ld.global.nc.v8.u32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
          : "=r"(b[u][0]), "=r"(b[u][1]), "=r"(b[u][2]), "=r"(b[u][3]), "=r"(b[u][4]),
            "=r"(b[u][5]), "=r"(b[u][6]), "=r"(b[u][7])
          : "l"(wp + 8 * (v0 + u)));
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      const uint4 a0 = hs[2 * (v0 + u)], a1 = hs[2 * (v0 + u) + 1];
      fma_lo(acc, a0.x, b[u][0]);
      fma_hi(acc, a0.x, b[u][0]);
      fma_lo(acc, a0.y, b[u][1]);
      fma_hi(acc, a0.y, b[u][1]);
      fma_lo(acc, a0.z, b[u][2]);
      fma_hi(acc, a0.z, b[u][2]);
      fma_lo(acc, a0.w, b[u][3]);
      fma_hi(acc, a0.w, b[u][3]);
      fma_lo(acc, a1.x, b[u][4]);
      fma_hi(acc, a1.x, b[u][4]);
      fma_lo(acc, a1.y, b[u][5]);
      fma_hi(acc, a1.y, b[u][5]);
      fma_lo(acc, a1.z, b[u][6]);
      fma_hi(acc, a1.z, b[u][6]);
      fma_lo(acc, a1.w, b[u][7]);
      fma_hi(acc, a1.w, b[u][7]);
    }
  }
  return acc;
}

__device__ __forceinline__ unsigned long long score_key(float v, int e) {
  v = (v == 0.0f) ? 0.0f : v;  // -0 and +0 are equal scores
  return (static_cast<unsigned long long>(order_bits(v)) << 32) |
         static_cast<unsigned long long>(0xffffffffu - static_cast<uint32_t>(e));
}

template <int NPL>
__global__ void __launch_bounds__(kScreenWarps * 32)
    screen_select_kernel(const __nv_bfloat16* __restrict__ h,
                         const __nv_bfloat16* __restrict__ w, float* __restrict__ z,
                         int k_splits, int64_t split_stride, const float* __restrict__ nw,
                         float g, const int32_t* __restrict__ kin, int T, int E, int d,
                         int k_max, int32_t* __restrict__ ids, float* __restrict__ alpha,
                         uint32_t* __restrict__ err, int wide) {
  extern __shared__ uint4 s_h[];  // [kScreenWarps][d / 8]: the warps' token rows
  __shared__ float s_z[kScreenWarps][32];
  __shared__ int32_t s_e[kScreenWarps][32];
  __shared__ int32_t s_c[kScreenWarps][32];
  grid_dep_wait();
  grid_dep_launch();
  const int wid = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t = blockIdx.x * kScreenWarps + wid;
  if (t >= T) return;
  const int kcap = k_max < E ? k_max : E;
  int kt = kin[t];
  if (kt < 1 || kt > kcap) {
    if (lane == 0) set_err(err, kErrKRange);
    kt = kt < 1 ? 1 : kcap;
  }
  const __nv_bfloat16* ht = h + static_cast<int64_t>(t) * d;
  uint4* hs = s_h + static_cast<int64_t>(wid) * (d / 8);
  // the token row into shared memory and ||h_t||_2, rounded up
  float ss = 0.f;
  for (int v = lane; v < d / 8; v += 32) {
    const uint4 q = reinterpret_cast<const uint4*>(ht)[v];
    hs[v] = q;
    const uint32_t wd[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float a = __uint_as_float(wd[i] << 16), b = __uint_as_float(wd[i] & 0xffff0000u);
      ss = fmaf(a, a, ss);
      ss = fmaf(b, b, ss);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  __syncwarp();  // the row in shared memory is visible to every lane
  const float nh = sqrtf(ss * (1.0f + 0x1p-10f)) * (1.0f + 0x1p-20f);
  // screen estimates and their intervals; L = k_t-th largest lower end
  float* zt = z + static_cast<int64_t>(t) * E;
  float zs[NPL], hi[NPL];
  unsigned long long key[NPL];
#pragma unroll
  for (int i = 0; i < NPL; ++i) {
    const int e = lane + 32 * i;
    zs[i] = 0.f;
    hi[i] = -INFINITY;
    key[i] = 0ull;
    if (e < E) {
      float v = zt[e];
      for (int s = 1; s < k_splits; ++s) v += zt[s * split_stride + e];
      const float del = g * nh * nw[e] * (1.0f + 0x1p-16f) + fabsf(v) * 0x1p-22f;
      zs[i] = v;
      hi[i] = v + del;
      key[i] = score_key(v - del, e);
    }
  }
  unsigned long long best = 0ull;
  for (int j = 0; j < kt; ++j) {
    best = key[0];
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
  }
  const float L = from_order_bits(static_cast<uint32_t>(best >> 32));
  // candidates: hi_e >= L, compacted into s_c (at most 32, else all experts)
  int m = 0;
#pragma unroll
  for (int i = 0; i < NPL; ++i) {
    const bool c = hi[i] >= L;
    const uint32_t mask = __ballot_sync(0xffffffffu, c);
    const int pos = m + __popc(mask & ((1u << lane) - 1u));
    if (c && pos < 32) s_c[wid][pos] = lane + 32 * i;
    m += __popc(mask);
  }
  __syncwarp();
  // every screen estimate stays in z, then the recomputed scores replace the
  // candidates' entries
#pragma unroll
  for (int i = 0; i < NPL; ++i)
    if (lane + 32 * i < E) zt[lane + 32 * i] = zs[i];
  __syncwarp();  // the estimates land before any lane overwrites a candidate's
  unsigned long long ck[NPL];
  if (m <= 32) {
    unsigned long long mine = 0ull;
    if (lane < m) {
      const int e = s_c[wid][lane];
      const float v = (wide ? chain_bf16_wide(hs, w + static_cast<int64_t>(e) * d, d)
                    : chain_bf16(hs, w + static_cast<int64_t>(e) * d, d));
      zt[e] = v;
      mine = score_key(v, e);
    }
#pragma unroll
    for (int i = 0; i < NPL; ++i) ck[i] = i == 0 ? mine : 0ull;
  } else {
#pragma unroll
    for (int i = 0; i < NPL; ++i) {
      const int e = lane + 32 * i;
      ck[i] = 0ull;
      if (e < E) {
        const float v = (wide ? chain_bf16_wide(hs, w + static_cast<int64_t>(e) * d, d)
                    : chain_bf16(hs, w + static_cast<int64_t>(e) * d, d));
        zt[e] = v;
        ck[i] = score_key(v, e);
      }
    }
  }
  // TopK over the recomputed scores (same keys and tie rule as select_token)
  for (int j = 0; j < kt; ++j) {
    unsigned long long b = ck[0];
#pragma unroll
    for (int i = 1; i < NPL; ++i) b = ck[i] > b ? ck[i] : b;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const unsigned long long other = __shfl_xor_sync(0xffffffffu, b, o);
      b = other > b ? other : b;
    }
#pragma unroll
    for (int i = 0; i < NPL; ++i)
      if (ck[i] == b) ck[i] = 0ull;
    if (lane == 0) {
      s_e[wid][j] = static_cast<int>(0xffffffffu - static_cast<uint32_t>(b & 0xffffffffull));
      s_z[wid][j] = from_order_bits(static_cast<uint32_t>(b >> 32));
    }
  }
  __syncwarp();
  const float zmax = s_z[wid][0];
  const float mine = lane < kt ? expf(s_z[wid][lane] - zmax) : 0.f;
  float sel = mine;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) sel += __shfl_xor_sync(0xffffffffu, sel, o);
  for (int j = lane; j < k_max; j += 32) {
    const int64_t o = static_cast<int64_t>(t) * k_max + j;
    if (j < kt) {
      ids[o] = s_e[wid][j];
      alpha[o] = mine / sel;
    } else {
      ids[o] = -1;
      alpha[o] = 0.f;
    }
  }
}

// ---- batched screen recheck (bf16, up to 256 experts) -----------------------
// The screen of screen_select_kernel for many tokens, where one warp per
// token streams each candidate's expert row from L2 one lane at a time.  A
// CTA owns a block of tokens (BatchCfg: 32 tokens and three CTAs per SM up
// to 64 experts; at 32 x 1024 tokens 1024 CTAs spread evenly over the SMs,
// where 64-token CTAs, two per SM, left some SMs idle for half of the
// kernel and 16-token CTAs stream the expert rows too often):
//   1. screening (8 warps, the CTA's tokens in turn, up to four tokens'
//      rounds interleaved):
//      from the tensor-core estimates z~ and the row norms (the score GEMM's
//      sums of squares, ||w_e|| from wnorm_kernel) the interval z~ -/+ del
//      of every (token, expert), the k_t-th largest lower end L, and the
//      candidates (upper end >= L) as a per-token bit mask; a prefix over
//      the tokens lays the (token, expert) candidate pairs out in shared
//      memory;
//   2. chains: a producer warp streams 64-k chunks of the CTA's token rows
//      and of the 32 NPL expert rows through a TMA ring (128-byte
//      swizzle); each compute thread advances the canonical fma chain of two
//      candidate pairs over the chunk, the pairs laid out so that a quarter
//      warp's expert rows fall in distinct bank groups (more than 512 pairs:
//      the rows are streamed again for the next 512);
//   3. selection (a warp per token): TopK over the candidates' exact
//      scores by rank counting, with the keys and tie rule of select_kernel,
//      the weights with its arithmetic (the same bits), and the exact scores
//      into z.
constexpr int kBatchCompute = 256;            // 8 compute warps
constexpr int kBatchThreads = kBatchCompute + 32;  // + the producer warp
constexpr int kBatchSlots = 2 * kBatchCompute;     // candidate pairs per pass
constexpr uint64_t kBatchWaitNs = 2000000000ull;
constexpr uint64_t kBatchDrainNs = 1000000000ull;
// NPL groups of 32 experts: every lane of a screening warp holds NPL of a
// token's experts, and every stage holds the 32 NPL expert rows.  Up to 64
// experts (NPL 2): 32 tokens per CTA, three CTAs per SM, four tokens'
// rounds interleaved per warp; up to 256 (NPL 8): 16 tokens per CTA, a
// 2-stage ring, two CTAs per SM, one token at a time (LLaDA2.0-mini layer
// 0.553 ms with 32 tokens and one CTA per SM, 0.558 with 16 and one, 0.546
// with 16 and two).
template <int NPL>
struct BatchCfg {
  static constexpr int kT = NPL <= 2 ? 32 : 16;       // tokens per CTA
  static constexpr int kE = 32 * NPL;                 // expert rows per stage
  static constexpr int kStages = NPL <= 2 ? 4 : 2;
  static constexpr int kMinCtas = NPL <= 2 ? 3 : 2;   // co-resident CTAs per SM
  static constexpr int kGroup = NPL <= 2 ? 4 : 1;     // tokens whose rounds interleave
  static constexpr int kIdBits = NPL <= 2 ? 6 : 8;    // expert index bits of a key
  static constexpr uint32_t kTokBytes = kT * 128;
  static constexpr uint32_t kStageBytes = kTokBytes + kE * 128;
  static_assert(kT % 8 == 0 && kT <= 64, "whole swizzle atoms; the prefix's 64 lanes");
};
template <int NPL>
struct BatchSmem {
  static constexpr int kT = BatchCfg<NPL>::kT;
  uint64_t full[BatchCfg<NPL>::kStages];
  uint64_t empty[BatchCfg<NPL>::kStages];
  uint32_t mask[kT][NPL];
  int32_t cnt[kT];
  int32_t kt[kT];
  int32_t off[kT + 1];
  float sel_z[8][32];
  int32_t sel_e[8][32];
  volatile int abort;
  uint16_t pair[kT * 32 * NPL];                 // (token << 8) | expert
  uint16_t slot[kT * 32 * NPL];                 // chain slot -> pair (0xffff: none)
  float zc[kT * 32 * NPL];                      // exact scores of the pairs
};
template <int NPL>
constexpr size_t batch_smem_bytes() {
  return 1024 + BatchCfg<NPL>::kStages * BatchCfg<NPL>::kStageBytes + sizeof(BatchSmem<NPL>);
}
static_assert(batch_smem_bytes<8>() <= 227 * 1024, "one CTA per SM at 256 experts");

// 16 bytes of shared memory.  The "memory" clobber keeps every such read
// between the stage's mbarrier wait and its release (both asm statements
// with the same clobber): without it the compiler may move a read of a ring
// stage above the wait that makes the TMA data visible.
__device__ __forceinline__ uint4 lds128(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(addr)
               : "memory");
  return v;
}
// Row r of a 128-byte-swizzled box of 128-byte rows at a 1024-aligned
// address: the 16-byte chunk q sits at r * 128 + ((q ^ (r & 7)) << 4), i.e.
// at (base + r * 128 + ((r & 7) << 4)) ^ (q << 4) (bits 4-6 of the row base
// hold r & 7); swz_row gives the part before the XOR.
__device__ __forceinline__ uint32_t swz_row(int r) {
  return static_cast<uint32_t>(r * 128 + ((r & 7) << 4));
}
__device__ __forceinline__ void chain8(float& acc, const uint4& a, const uint4& b) {
  fma_lo(acc, a.x, b.x);
  fma_hi(acc, a.x, b.x);
  fma_lo(acc, a.y, b.y);
  fma_hi(acc, a.y, b.y);
  fma_lo(acc, a.z, b.z);
  fma_hi(acc, a.z, b.z);
  fma_lo(acc, a.w, b.w);
  fma_hi(acc, a.w, b.w);
}
// 32-bit screening key for at most 2^B experts: the order bits of an
// interval's lower end with the low B bits replaced by 2^B - 1 - e (so no
// two experts tie, and the lower index wins among equal truncated values).
// Truncation is monotone, so the k-th largest key's value part is the
// truncated k-th largest lower end: the threshold it gives is never above
// the exact one and the candidates are a superset of the exact candidates.
// 0 stays free for "removed" (only a negative NaN could map there).
template <int B>
__device__ __forceinline__ uint32_t screen_key(float v, int e) {
  constexpr uint32_t m = (1u << B) - 1u;
  v = (v == 0.0f) ? 0.0f : v;
  const uint32_t k = (order_bits(v) & ~m) | (m - static_cast<uint32_t>(e));
  return k != 0u ? k : 1u;
}

template <int NPL>
__global__ void __launch_bounds__(kBatchThreads, BatchCfg<NPL>::kMinCtas)
    screen_batch_kernel(const __grid_constant__ CUtensorMap map_h,
                        const __grid_constant__ CUtensorMap map_w, float* __restrict__ z,
                        const float* __restrict__ hss, const float* __restrict__ nw, float g,
                        const int32_t* __restrict__ kin, int T, int E, int d, int k_max,
                        int32_t* __restrict__ ids, float* __restrict__ alpha,
                        uint32_t* __restrict__ err) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* ring = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  using Cf = BatchCfg<NPL>;
  constexpr int kBatchT = Cf::kT;
  constexpr int kBatchStages = Cf::kStages;
  constexpr uint32_t kBatchTokBytes = Cf::kTokBytes;
  constexpr int kGroup = Cf::kGroup;
  constexpr uint32_t kStageBytes = Cf::kStageBytes;
  constexpr uint32_t kIdMask = (1u << Cf::kIdBits) - 1u;
  BatchSmem<NPL>& sm =
      *reinterpret_cast<BatchSmem<NPL>*>(ring + kBatchStages * kStageBytes);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t0 = blockIdx.x * kBatchT;
  const int nt = min(kBatchT, T - t0);
  const int kcap = k_max < E ? k_max : E;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kBatchStages; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], kBatchCompute / 32);
    }
    sm.abort = 0;
    fence_mbar_init();
  }
  grid_dep_wait();
  grid_dep_launch();
  // ---- 1. screening: candidate masks, kGroup tokens' rounds interleaved ----
  if (warp < 8) {
    float nwj[NPL];  // the norms of this lane's experts lane + 32 j
#pragma unroll
    for (int j = 0; j < NPL; ++j) nwj[j] = lane + 32 * j < E ? nw[lane + 32 * j] : 0.f;
    for (int g0 = 0; g0 < kBatchT / 8; g0 += kGroup) {
      float zv[kGroup][NPL], hs[kGroup];
      int kt[kGroup];
#pragma unroll
      for (int i = 0; i < kGroup; ++i) {  // every load of the group first
        // a warp's last group is partial when kBatchT / 8 is not a multiple
        // of kGroup
        const int tl = warp * (kBatchT / 8) + g0 + i;
        const int t = t0 + tl;
        const bool ok = g0 + i < kBatchT / 8 && tl < nt;
        kt[i] = ok ? kin[t] : 1;
        hs[i] = ok ? hss[t] : 0.f;
        const float* zt = z + static_cast<int64_t>(ok ? t : 0) * E;
#pragma unroll
        for (int j = 0; j < NPL; ++j)
          zv[i][j] = ok && lane + 32 * j < E ? zt[lane + 32 * j] : 0.f;
      }
      // 32-bit keys: one shuffle per step of the rounds' warp maximum
      uint32_t key[kGroup][NPL], best[kGroup];
      float hi[kGroup][NPL];
      int rounds = 0;
#pragma unroll
      for (int i = 0; i < kGroup; ++i) {
        if (kt[i] < 1 || kt[i] > kcap) {
          const int tl = warp * (kBatchT / 8) + g0 + i;
          if (lane == 0 && g0 + i < kBatchT / 8 && tl < nt) set_err(err, kErrKRange);
          kt[i] = kt[i] < 1 ? 1 : kcap;
        }
        rounds = max(rounds, kt[i]);
        const float nh = sqrtf(hs[i] * (1.0f + 0x1p-10f)) * (1.0f + 0x1p-20f);
#pragma unroll
        for (int j = 0; j < NPL; ++j) {
          const int e = lane + 32 * j;
          hi[i][j] = -INFINITY;
          key[i][j] = 0u;
          if (e < E) {
            const float v = zv[i][j];
            const float del = g * nh * nwj[j] * (1.0f + 0x1p-16f) + fabsf(v) * 0x1p-22f;
            hi[i][j] = v + del;
            key[i][j] = screen_key<Cf::kIdBits>(v - del, e);
          }
        }
        best[i] = 0u;
      }
      for (int r = 0; r < rounds; ++r) {
        uint32_t b[kGroup];
#pragma unroll
        for (int i = 0; i < kGroup; ++i) {
          b[i] = key[i][0];
#pragma unroll
          for (int j = 1; j < NPL; ++j) b[i] = max(b[i], key[i][j]);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1)
#pragma unroll
          for (int i = 0; i < kGroup; ++i)
            b[i] = max(b[i], __shfl_xor_sync(0xffffffffu, b[i], o));
#pragma unroll
        for (int i = 0; i < kGroup; ++i) {
          if (r < kt[i]) {
            best[i] = b[i];
#pragma unroll
            for (int j = 0; j < NPL; ++j)
              if (key[i][j] == b[i]) key[i][j] = 0u;
          }
        }
      }
#pragma unroll
      for (int i = 0; i < kGroup; ++i) {
        if (g0 + i >= kBatchT / 8) break;  // the next warp's token
        const int tl = warp * (kBatchT / 8) + g0 + i;
        const float L = from_order_bits(best[i] & ~kIdMask);
        int c = 0;
#pragma unroll
        for (int j = 0; j < NPL; ++j) {
          const uint32_t m = __ballot_sync(0xffffffffu, tl < nt && hi[i][j] >= L);
          if (lane == 0) sm.mask[tl][j] = m;
          c += __popc(m);
        }
        if (lane == 0) {
          sm.cnt[tl] = c;
          sm.kt[tl] = tl < nt ? kt[i] : 0;
        }
      }
    }
  }
  __syncthreads();
  if (warp == 0) {  // exclusive prefix of the candidate counts
    int a = lane < kBatchT ? sm.cnt[lane] : 0;
    int b = lane + 32 < kBatchT ? sm.cnt[lane + 32] : 0;
    int ia = a, ib = b;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int va = __shfl_up_sync(0xffffffffu, ia, o);
      const int vb = __shfl_up_sync(0xffffffffu, ib, o);
      if (lane >= o) {
        ia += va;
        ib += vb;
      }
    }
    const int tot_a = __shfl_sync(0xffffffffu, ia, 31);
    if (lane < kBatchT) sm.off[lane] = ia - a;
    if (lane + 32 < kBatchT) sm.off[lane + 32] = tot_a + ib - b;
    if (lane == 31) sm.off[kBatchT] = tot_a + ib;  // the total
  }
  __syncthreads();
  if (warp < 8) {  // the (token, expert) pairs in token order, experts ascending
    for (int i = 0; i < kBatchT / 8; ++i) {
      const int tl = warp * (kBatchT / 8) + i;
      const uint32_t below = (1u << lane) - 1u;
      int pos = sm.off[tl];
#pragma unroll
      for (int j = 0; j < NPL; ++j) {
        const uint32_t m = sm.mask[tl][j];
        if ((m >> lane) & 1u)
          sm.pair[pos + __popc(m & below)] = static_cast<uint16_t>((tl << 8) | (lane + 32 * j));
        pos += __popc(m);
      }
    }
  }
  __syncthreads();
  const int npairs = sm.off[kBatchT];
  // Chain slots: each run of 32 pairs is reordered so that the 8 lanes of a
  // quarter warp read expert rows of distinct swizzle classes (e & 7): a
  // 16-byte shared load is served a quarter warp per wavefront, and rows of
  // one class share a bank group.  The pairs are sorted by class within the
  // run and dealt to the quarters in turn (sorted position i -> lane
  // 8 (i % 4) + i / 4).
  if (warp < 8) {
    for (int base = warp * 32; base < npairs; base += 8 * 32) {
      const int idx = base + lane;
      const bool valid = idx < npairs;
      const int cls = valid ? (sm.pair[idx] & 7) : 8;
      int pos = 0;
#pragma unroll
      for (int c = 0; c <= 8; ++c) {
        const uint32_t mc = __ballot_sync(0xffffffffu, cls == c);
        if (c < cls) pos += __popc(mc);
        if (c == cls) pos += __popc(mc & ((1u << lane) - 1u));
      }
      sm.slot[base + 8 * (pos & 3) + (pos >> 2)] = valid ? static_cast<uint16_t>(idx) : 0xffff;
    }
  }
  __syncthreads();
  const int nslots = (npairs + 31) & ~31;
  const int passes = (nslots + kBatchSlots - 1) / kBatchSlots;
  const int nch = d / 64;
  // ---- 2. the chains ----
  if (warp == 8) {
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0, issued = 0, issued_phase = 0;
      bool ok = true;
      for (int ps = 0; ps < passes && ok; ++ps) {
        for (int c = 0; c < nch; ++c) {
          if (!mbar_wait(&sm.empty[stage], phase ^ 1u, &sm.abort, kBatchWaitNs)) {
            ok = false;
            break;
          }
          const uint32_t fb = smem_addr(&sm.full[stage]);
          uint8_t* st = ring + stage * kStageBytes;
          mbar_arrive_tx(fb, kStageBytes);
          tma_tile_2d(smem_addr(st), &map_h, c * 64, t0, fb);
          tma_tile_2d(smem_addr(st + kBatchTokBytes), &map_w, c * 64, 0, fb);
          issued |= 1u << stage;
          issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
          if (++stage == kBatchStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok) {
        set_err(err, kErrTimeout);
        sm.abort = 1;
      }
      if (sm.abort) {  // every issued copy lands before the CTA exits
        for (int s = 0; s < kBatchStages; ++s)
          if (issued & (1u << s))
            mbar_wait(&sm.full[s], (issued_phase >> s) & 1u, nullptr, kBatchDrainNs);
      }
    }
  } else {
    const uint32_t ring_s = smem_addr(ring);
    int stage = 0;
    uint32_t phase = 0;
    bool ok = true;
    for (int ps = 0; ps < passes && ok; ++ps) {
      const int s0 = ps * kBatchSlots + threadIdx.x, s1 = s0 + kBatchCompute;
      const int p0 = s0 < nslots ? sm.slot[s0] : 0xffff;
      const int p1 = s1 < nslots ? sm.slot[s1] : 0xffff;
      const uint32_t q0 = p0 != 0xffff ? sm.pair[p0] : 0u;
      const uint32_t q1 = p1 != 0xffff ? sm.pair[p1] : 0u;
      // row bases inside a stage (the swizzle is an XOR on bits 4-6)
      const uint32_t ta0 = swz_row(q0 >> 8), ea0 = kBatchTokBytes + swz_row(q0 & 255);
      const uint32_t ta1 = swz_row(q1 >> 8), ea1 = kBatchTokBytes + swz_row(q1 & 255);
      // the second slot only where a lane of the warp has a pair for it
      const bool two = __any_sync(0xffffffffu, p1 != 0xffff);
      float acc0 = 0.f, acc1 = 0.f;
      for (int c = 0; c < nch; ++c) {
        if (!__all_sync(0xffffffffu,
                        mbar_wait(&sm.full[stage], phase, &sm.abort, kBatchWaitNs))) {
          ok = false;
          break;
        }
        const uint32_t sb = ring_s + stage * kStageBytes;
        const uint32_t h0 = sb + ta0, w0 = sb + ea0, h1 = sb + ta1, w1 = sb + ea1;
        if (two) {
          uint4 a0 = lds128(h0), b0 = lds128(w0), a1 = lds128(h1), b1 = lds128(w1);
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            uint4 na0, nb0, na1, nb1;
            if (q + 1 < 8) {
              const uint32_t x = static_cast<uint32_t>((q + 1) << 4);
              na0 = lds128(h0 ^ x);
              nb0 = lds128(w0 ^ x);
              na1 = lds128(h1 ^ x);
              nb1 = lds128(w1 ^ x);
            }
            chain8(acc0, a0, b0);
            chain8(acc1, a1, b1);
            if (q + 1 < 8) {
              a0 = na0;
              b0 = nb0;
              a1 = na1;
              b1 = nb1;
            }
          }
        } else {
          uint4 a0 = lds128(h0), b0 = lds128(w0);
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            uint4 na0, nb0;
            if (q + 1 < 8) {
              const uint32_t x = static_cast<uint32_t>((q + 1) << 4);
              na0 = lds128(h0 ^ x);
              nb0 = lds128(w0 ^ x);
            }
            chain8(acc0, a0, b0);
            if (q + 1 < 8) {
              a0 = na0;
              b0 = nb0;
            }
          }
        }
        fence_proxy_async_smem();  // the reads above, before the next TMA fill
        __syncwarp();
        if (lane == 0) mbar_arrive_local(smem_addr(&sm.empty[stage]));
        if (++stage == kBatchStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
      if (ok) {
        if (p0 != 0xffff) sm.zc[p0] = acc0;
        if (p1 != 0xffff) sm.zc[p1] = acc1;
      }
    }
    if (!ok && lane == 0) {
      set_err(err, kErrTimeout);
      sm.abort = 1;
    }
  }
  __syncthreads();
  if (sm.abort) return;
  // ---- 3. selection over the candidates' exact scores ----
  // A warp per token: lane l takes candidates l + 32 j, keys as in
  // select_kernel (score, then the lower expert index); a candidate's rank is
  // the number of the token's candidates with a larger key, and the k_t
  // candidates of rank < k_t go to slot rank (the TopK in rank order).
  if (warp < 8) {
    for (int i = 0; i < kBatchT / 8; ++i) {
      const int tl = warp * (kBatchT / 8) + i;
      if (tl >= nt) continue;
      const int t = t0 + tl;
      const int off = sm.off[tl], m = sm.cnt[tl], kt = sm.kt[tl];
      const int nj = (m + 31) / 32;  // candidate groups of 32 in use
      float* zt = z + static_cast<int64_t>(t) * E;
      unsigned long long key[NPL];
      int ex[NPL];
#pragma unroll
      for (int j = 0; j < NPL; ++j) {
        const int idx = lane + 32 * j;
        key[j] = 0ull;
        ex[j] = 0;
        if (idx < m) {
          ex[j] = sm.pair[off + idx] & 255;
          const float v = sm.zc[off + idx];
          zt[ex[j]] = v;
          key[j] = score_key(v, ex[j]);
        }
      }
      // every candidate's key in shared memory (the token's zc slots hold
      // the scores; the keys are rebuilt from them), then the ranks
      int rank[NPL];
#pragma unroll
      for (int j = 0; j < NPL; ++j) rank[j] = 0;
      for (int o = 0; o < m; ++o) {
        const unsigned long long ko =
            score_key(sm.zc[off + o], sm.pair[off + o] & 255);  // broadcast reads
#pragma unroll
        for (int j = 0; j < NPL; ++j)
          if (j < nj) rank[j] += ko > key[j];
      }
#pragma unroll
      for (int j = 0; j < NPL; ++j) {
        if (lane + 32 * j < m && rank[j] < kt) {
          sm.sel_e[warp][rank[j]] = ex[j];
          sm.sel_z[warp][rank[j]] = from_order_bits(static_cast<uint32_t>(key[j] >> 32));
        }
      }
      __syncwarp();
      const float zmax = sm.sel_z[warp][0];
      const float mine = lane < kt ? expf(sm.sel_z[warp][lane] - zmax) : 0.f;
      float sel = mine;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) sel += __shfl_xor_sync(0xffffffffu, sel, o);
      for (int j = lane; j < k_max; j += 32) {
        const int64_t o = static_cast<int64_t>(t) * k_max + j;
        if (j < kt) {
          ids[o] = sm.sel_e[warp][j];
          alpha[o] = mine / sel;
        } else {
          ids[o] = -1;
          alpha[o] = 0.f;
        }
      }
      __syncwarp();
    }
  }
}

template <int LY, int TM, int TN, int WT, int WE, int S, int KC = 32>
cudaError_t launch_logits_mx(const __nv_bfloat16* h, const __nv_bfloat16* w, int T,
                             int d, int E, float* z, uint32_t* zw, int nz, cudaStream_t s) {
  using C = MxCfg<LY, TM, TN, WT, WE, S, KC>;
  auto kern = logits_mx_kernel<LY, TM, TN, WT, WE, S, KC>;
  if (C::kSmem > 48 * 1024) {
    const cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmem);
    if (e != cudaSuccess) return e;
  }
  const dim3 g((T + C::BT - 1) / C::BT, (E + C::BE - 1) / C::BE);
  kern<<<g, C::NT, C::kSmem, s>>>(h, w, T, d, E, z, zw, nz);
  return cudaGetLastError();
}

// fp32 inputs: the widened-buffer tiles when they fill most SMs without
// overhanging the expert count; otherwise the short-batch kernel with the
// largest token tile that still fills most SMs.
cudaError_t logits_dispatch(const float* h, const float* w, int T, int d, int E,
                            float* z, uint32_t* zw, int nz, int num_sms, cudaStream_t s) {
  auto grid_for = [&](int bt, int be) {
    return static_cast<int64_t>((T + bt - 1) / bt) * ((E + be - 1) / be);
  };
  const int64_t want = (num_sms * 4) / 5;
  if (E >= 128 && grid_for(64, 128) >= want)  // TM 4, TN 8, 2 x 4 warps
    return launch_logits_tile<float, 4, 8, 2, 4>(h, w, T, d, E, z, zw, nz, s);
  if (grid_for(32, 64) >= want) return launch_logits_short<float, 4>(h, w, T, d, E, z, zw, nz, s);
  if (grid_for(16, 64) >= want) return launch_logits_short<float, 2>(h, w, T, d, E, z, zw, nz, s);
  return launch_logits_short<float, 1>(h, w, T, d, E, z, zw, nz, s);
}

// The score kernels are launched without programmatic serialization: with a
// tile count of one or two CTAs per SM, CTAs placed early on the SMs that a
// wide predecessor (the previous layer's combine) frees first pile up there,
// and the unbalanced placement cost up to 100 us at 4096 x 256 scores on
// GB300.  They still clear the header and let the next kernel launch early.
//
// bf16 inputs: mixed-precision fma tiles, chosen by the number of chains
// T x E per SM (measured on GB300 over T = 256 .. 65536, E = 64 and 256).
// Few chains: small thread tiles so every SM gets warps; many chains: 4 x 8
// or 4 x 4 thread tiles, which need fewer operand reads per fma.
cudaError_t logits_dispatch(const __nv_bfloat16* h, const __nv_bfloat16* w, int T,
                            int d, int E, float* z, uint32_t* zw, int nz, uint32_t* err,
                            int num_sms, cudaStream_t s, const L2Prefetch& pf) {
  const int64_t per_sm = static_cast<int64_t>(T) * E / (num_sms > 0 ? num_sms : 1);
  // whole rows resident: 16 x 32 tiles, one CTA of 8 warps per SM (2 x 1
  // chains per thread), for about 300-640 chains per SM (1024 x 64 scores:
  // 20.8 -> 18.1 us; 8 warps of 2 x 1 instead of 4 of 2 x 2: step -0.6 us;
  // fewer chains favour the ring kernel's smaller tiles, more chains need a
  // second wave)
  using Res = ResCfg<4, 2, 1, 2, 4>;
  if (per_sm > 300 && per_sm <= 640 && d % kResChunkK == 0 &&
      d / kResChunkK <= kResMaxChunks && Res::smem(d) <= 227 * 1024)
    return launch_logits_res<4, 2, 1, 2, 4>(h, w, T, d, E, z, zw, nz, err, pf, s);
  if (per_sm <= 216) return launch_logits_mx<4, 1, 1, 4, 1, 8>(h, w, T, d, E, z, zw, nz, s);
  if (per_sm <= 1080) return launch_logits_mx<4, 1, 2, 4, 1, 8>(h, w, T, d, E, z, zw, nz, s);
  if (per_sm <= 4300) return launch_logits_mx<4, 2, 2, 2, 2, 4, 64>(h, w, T, d, E, z, zw, nz, s);
  if (per_sm <= 10000) return launch_logits_mx<8, 4, 8, 2, 2, 3, 64>(h, w, T, d, E, z, zw, nz, s);
  if (per_sm <= 20000) return launch_logits_mx<8, 4, 4, 2, 2, 3, 64>(h, w, T, d, E, z, zw, nz, s);
  return launch_logits_mx<8, 4, 8, 2, 2, 4>(h, w, T, d, E, z, zw, nz, s);
}

}  // namespace

cudaError_t launch_router_logits(int dtype, const void* hidden,
                                 const void* w_router, int T, int d, int E,
                                 float* z, uint32_t* zero_words, int n_zero,
                                 uint32_t* err, int num_sms, cudaStream_t stream,
                                 const L2Prefetch& pf) {
  if (T == 0) return cudaSuccess;
  if (dtype == 0)
    return logits_dispatch(static_cast<const float*>(hidden),
                           static_cast<const float*>(w_router), T, d, E, z,
                           zero_words, n_zero, num_sms, stream);
  return logits_dispatch(static_cast<const __nv_bfloat16*>(hidden),
                         static_cast<const __nv_bfloat16*>(w_router), T, d, E,
                         z, zero_words, n_zero, err, num_sms, stream, pf);
}

cudaError_t launch_router_wnorm(const __nv_bfloat16* w, int E, int d, float* nw,
                                uint32_t* zero_words, int n_zero, cudaStream_t stream) {
  // plain launch: the first kernel of the forward
  wnorm_kernel<<<(E + 7) / 8, 256, 0, stream>>>(w, E, d, nw, zero_words, n_zero);
  return cudaGetLastError();
}

cudaError_t launch_router_screen_select(const __nv_bfloat16* h, const __nv_bfloat16* w,
                                        float* z, int k_splits, int64_t split_stride,
                                        const float* nw, const int32_t* k, int T, int E,
                                        int d, int k_max, int32_t* ids, float* alpha,
                                        uint32_t* err, cudaStream_t stream) {
  if (T == 0) return cudaSuccess;
  if (d % kScreenDMultiple != 0 || E > 1024 || k_splits < 1) return cudaErrorInvalidValue;
  const size_t smem = static_cast<size_t>(kScreenWarps) * d * 2;  // bf16 token rows
  const double u = 1.0 / 16777216.0;
  const double gamma = d * u / (1.0 - d * u);
  // chain bound + tensor-core allowance + one rounding per split-K slice
  const float g = static_cast<float>((gamma + 1.0 / 4096.0 + (k_splits + 1) * u) * (1.0 + 1e-3));
  const dim3 grid((T + kScreenWarps - 1) / kScreenWarps), block(kScreenWarps * 32);
  // 32-byte row loads when every expert row starts on a 32-byte boundary
  const int wide = (reinterpret_cast<uintptr_t>(w) % 32 == 0 && d % 32 == 0) ? 1 : 0;
#define RX_SCREEN(N)                                                                     \
  (smem > 48 * 1024 && cudaFuncSetAttribute(screen_select_kernel<N>,                     \
                                            cudaFuncAttributeMaxDynamicSharedMemorySize, \
                                            static_cast<int>(smem)) != cudaSuccess)      \
      ? cudaErrorInvalidValue                                                            \
      : launch_pdl(screen_select_kernel<N>, grid, block, smem, stream, h, w, z, k_splits, \
                   split_stride, nw, g, k, T, E, d, k_max, ids, alpha, err, wide)
  if (E <= 32) return RX_SCREEN(1);
  if (E <= 64) return RX_SCREEN(2);
  if (E <= 128) return RX_SCREEN(4);
  if (E <= 256) return RX_SCREEN(8);
  if (E <= 512) return RX_SCREEN(16);
  return RX_SCREEN(32);
#undef RX_SCREEN
}

cudaError_t launch_router_screen_batch(const CUtensorMap* map_h, const CUtensorMap* map_w,
                                       float* z, const float* hss, const float* nw,
                                       const int32_t* k, int T, int E, int d, int k_max,
                                       int32_t* ids, float* alpha, uint32_t* err,
                                       cudaStream_t stream) {
  if (T == 0) return cudaSuccess;
  if (E > 256 || d % 64 != 0 || d < 64 || k_max > 32) return cudaErrorInvalidValue;
  const double u = 1.0 / 16777216.0;
  const double gamma = d * u / (1.0 - d * u);
  // chain bound + tensor-core allowance + the score's own rounding (one K slice)
  const float g = static_cast<float>((gamma + 1.0 / 4096.0 + 2 * u) * (1.0 + 1e-3));
  auto go = [&](auto kernel, size_t smem, int rows) -> cudaError_t {
    const cudaError_t e =
        cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const dim3 grid((T + rows - 1) / rows), block(kBatchThreads);
    return launch_pdl(kernel, grid, block, smem, stream, *map_h, *map_w, z, hss, nw, g, k, T,
                      E, d, k_max, ids, alpha, err);
  };
  // map_h's box is screen_batch_token_rows(E) rows high, map_w's
  // screen_batch_expert_rows(E)
  if (E <= 64) return go(screen_batch_kernel<2>, batch_smem_bytes<2>(), BatchCfg<2>::kT);
  return go(screen_batch_kernel<8>, batch_smem_bytes<8>(), BatchCfg<8>::kT);
}

int screen_batch_token_rows(int E) { return E <= 64 ? BatchCfg<2>::kT : BatchCfg<8>::kT; }
int screen_batch_expert_rows(int E) { return E <= 64 ? BatchCfg<2>::kE : BatchCfg<8>::kE; }

cudaError_t launch_router_select_rule(const float* z, int T, int E, int k_hi, int k_lo,
                                      int rule, float thr, int k_max, bool renorm,
                                      int32_t* k_out, unsigned long long* k_sum,
                                      int32_t* ids, float* alpha, cudaStream_t stream) {
  if (T == 0) return cudaSuccess;
  if (rule != 1 && rule != 2) return cudaErrorInvalidValue;
  const dim3 grid((T + kSelWarps - 1) / kSelWarps);
  const dim3 block(kSelWarps * 32);
  const int r = renorm ? 1 : 0;
#define RX_SEL_RULE(N)                                                                   \
  launch_pdl(select_rule_kernel<N>, grid, block, 0, stream, z, T, E, k_hi, k_lo, rule, thr, \
             k_max, r, k_out, k_sum, ids, alpha)
  if (E <= 32) return RX_SEL_RULE(1);
  if (E <= 64) return RX_SEL_RULE(2);
  if (E <= 128) return RX_SEL_RULE(4);
  if (E <= 256) return RX_SEL_RULE(8);
  if (E <= 512) return RX_SEL_RULE(16);
  return RX_SEL_RULE(32);
#undef RX_SEL_RULE
}

cudaError_t launch_router_select(const float* z, const int32_t* k, int T,
                                 int E, int k_max, bool renorm, int32_t* ids,
                                 float* alpha, uint32_t* err,
                                 cudaStream_t stream) {
  if (T == 0) return cudaSuccess;
  const dim3 grid((T + kSelWarps - 1) / kSelWarps);
  const dim3 block(kSelWarps * 32);
  const int r = renorm ? 1 : 0;
  cudaError_t e;
  if (E <= 32)
    e = launch_pdl(select_kernel<1>, grid, block, 0, stream, z, k, T, E, k_max, r, ids, alpha, err);
  else if (E <= 64)
    e = launch_pdl(select_kernel<2>, grid, block, 0, stream, z, k, T, E, k_max, r, ids, alpha, err);
  else if (E <= 128)
    e = launch_pdl(select_kernel<4>, grid, block, 0, stream, z, k, T, E, k_max, r, ids, alpha, err);
  else if (E <= 256)
    e = launch_pdl(select_kernel<8>, grid, block, 0, stream, z, k, T, E, k_max, r, ids, alpha, err);
  else if (E <= 512)
    e = launch_pdl(select_kernel<16>, grid, block, 0, stream, z, k, T, E, k_max, r, ids, alpha, err);
  else
    e = launch_pdl(select_kernel<32>, grid, block, 0, stream, z, k, T, E, k_max, r, ids, alpha, err);
  return e;
}

}  // namespace rx
