// budget.cu — per-token expert counts of one denoising forward (REFLEX,
// Sec. 4.2-4.3): Refinement-Role Budgeting (Eq. 5), Frontier-Guided Expert
// Reallocation with the Frontier-Progress Score (forecast, Eq. 6-8, Eq. 9),
// then the clip to [K_min, K_max] of the count set in Eq. 3.
//
// One CTA per sequence.  Pass 1 writes the role count of every token and
// gathers J_h (masked active-block tokens with history) with their scores in
// shared memory; pass 2 ranks J_h by (S desc, position asc) with an
// all-pairs rank count — the block holds a few dozen tokens (block length 32
// in Sec. 5.1), so the O(|J|^2) count is a few hundred compares per thread.
//
// The score is computed in fp32 with one rounding per operation, in a fixed
// order, and with an exp written here from Cody & Waite's argument reduction
// and a degree-7 Taylor polynomial, so that the ranking (an integer result)
// is reproducible bit for bit.  The ablations of App. C are options: other
// rank keys (F, P, c^{t-1}, 1 - c^{t-1}) and a seeded permutation of each
// sequence's final counts (Role-Shuffled RRB).
#include "common.cuh"
#include "internal.h"
#include "reflex.h"

namespace rx {
namespace {

constexpr int kThreads = 1024;  // one token per thread for sequences up to 1024
constexpr int kMaxJ = 4096;

__device__ __forceinline__ float sigmoid_cw(float x) {
  return __fdiv_rn(1.0f, __fadd_rn(1.0f, exp_cw(-x)));
}

// Rank key of a member of J_h from the two latest confidences (hist =
// number of observations available).  REFLEX_SIGNAL_FPS is the
// Frontier-Progress Score S = F * P (Eq. 6-8); the other keys are the
// single-signal ablations: F, P, c^{t-1}, 1 - c^{t-1}.
__device__ float rank_key(int signal, float c1, float c2, int hist, float theta, float w,
                          float v_ref, float tau) {
  if (signal == REFLEX_SIGNAL_CONFIDENCE) return c1;
  if (signal == REFLEX_SIGNAL_UNCERTAINTY) return __fsub_rn(1.0f, c1);
  const float v = hist >= 2 ? __fsub_rn(c1, c2) : 0.0f;
  const float half_w = __fmul_rn(w, 0.5f);
  const float vbar = fminf(fmaxf(v, -half_w), half_w);
  const float P =
      hist >= 2 ? sigmoid_cw(__fdiv_rn(__fsub_rn(v_ref, vbar), tau)) : 1.0f;
  if (signal == REFLEX_SIGNAL_PROGRESS) return P;
  const float chat = fminf(fmaxf(__fadd_rn(c1, vbar), 0.0f), 1.0f);
  const float x1 = __fdiv_rn(__fadd_rn(__fsub_rn(chat, theta), w), tau);
  const float x2 = __fdiv_rn(__fsub_rn(theta, chat), tau);
  const float F = __fmul_rn(sigmoid_cw(x1), sigmoid_cw(x2));
  if (signal == REFLEX_SIGNAL_FRONTIER) return F;
  return __fmul_rn(F, P);
}

// Role-shuffle key of the token at batch index pos: the high 32 bits of
// splitmix64 output number pos + 1 for the seed (Steele, Lea and Flood 2014:
// state advances by the golden gamma, output is Stafford's mix13 of it).
__device__ __forceinline__ uint32_t shuffle_key(uint64_t seed, int pos) {
  uint64_t z = seed + static_cast<uint64_t>(pos + 1) * 0x9e3779b97f4a7c15ull;
  z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ull;
  z = (z ^ (z >> 27)) * 0x94d049bb133111ebull;
  z ^= z >> 31;
  return static_cast<uint32_t>(z >> 32);
}

__device__ __forceinline__ int role_count(int dist, int k_base, int d_role) {
  return dist <= 1 ? k_base + d_role : (dist == 2 ? k_base : k_base - d_role);
}

__device__ __forceinline__ int clip(int k, int lo, int hi) {
  return k < lo ? lo : (k > hi ? hi : k);
}

__device__ __forceinline__ void budget_body(const float* __restrict__ conf1,
                                            const float* __restrict__ conf2,
                                            const uint8_t* __restrict__ hist_len,
                                            const uint8_t* __restrict__ masked,
                                            const int32_t* __restrict__ block_id,
                                            const int32_t* __restrict__ seq_off,
                                            const int32_t* __restrict__ active_block,
                                            int T, const AllocArgs& a,
                                            int32_t* __restrict__ k_out,
                                            unsigned long long* __restrict__ k_sum,
                                            uint32_t* __restrict__ err) {
  // J_h scores and positions; the role shuffle reuses the same 32 KB as
  // kMaxJ 64-bit sort words
  __shared__ __align__(16) uint64_t s_raw[kMaxJ];
  float* s_score = reinterpret_cast<float*>(s_raw);
  int32_t* s_tok = reinterpret_cast<int32_t*>(s_raw) + kMaxJ;
  __shared__ int s_nj;
  __shared__ unsigned long long s_sum;
  __shared__ uint32_t s_err;
  // With one sequence (one CTA) the sum and the error word are stored
  // outright at the end, so the caller needs no clearing; with several,
  // the host clears them and each CTA adds its share.
  const bool sole = gridDim.x == 1;
  const int s = blockIdx.x;
  const int lo = seq_off[s], hi = seq_off[s + 1];
  if (lo < 0 || hi > T || lo > hi) {  // malformed offsets: touch no count
    if (threadIdx.x == 0) {
      if (sole) {
        if (err) *err = kErrIndex;
        if (k_sum) *k_sum = 0ull;
      } else {
        set_err(err, kErrIndex);
      }
    }
    return;
  }
  int act = active_block[s];
  if (threadIdx.x == 0) {
    s_nj = 0;
    s_sum = 0ull;
    s_err = act < 1 ? kErrActive : 0u;
  }
  __syncthreads();
  const int k_cur = a.k_base + a.delta_role;
  unsigned long long my_sum = 0;
  // pass 1: role counts (Eq. 5) and J_h membership with scores (Eq. 6-8)
  for (int i = lo + threadIdx.x; i < hi; i += kThreads) {
    const int b = block_id[i];
    const int dist = act >= 1 ? abs(b - act) : 3;
    int k = role_count(dist, a.k_base, a.delta_role);
    const bool in_j = act >= 1 && b == act && masked[i] != 0 && hist_len[i] >= 1;
    if (in_j) {
      const int slot = atomicAdd(&s_nj, 1);
      if (slot < kMaxJ) {
        s_tok[slot] = i;
        s_score[slot] = rank_key(a.signal, conf1[i], conf2[i], hist_len[i], a.theta,
                                 a.w_cf, a.v_ref, a.tau);
        continue;  // written in pass 2
      }
      k = k_cur;  // over capacity: keeps K_cur (error flagged below)
    }
    k = clip(k, a.k_min, a.k_max);
    k_out[i] = k;
    my_sum += static_cast<unsigned long long>(k);
  }
  __syncthreads();
  const int nj_all = s_nj;
  const int nj = nj_all < kMaxJ ? nj_all : kMaxJ;
  if (nj_all > kMaxJ) {
    // too many to rank: every stored member keeps K_cur too
    if (threadIdx.x == 0) atomicOr(&s_err, kErrCapacity);
    for (int m = threadIdx.x; m < nj; m += kThreads) {
      const int k = clip(k_cur, a.k_min, a.k_max);
      k_out[s_tok[m]] = k;
      my_sum += static_cast<unsigned long long>(k);
    }
  } else {
    // pass 2: Eq. 9 groups from the rank of each member
    const int n = static_cast<int>(floorf(__fmul_rn(a.q, static_cast<float>(nj))));
    for (int m = threadIdx.x; m < nj; m += kThreads) {
      const float sm = s_score[m];
      const int tm = s_tok[m];
      int rank = 0;
      for (int j = 0; j < nj; ++j) {
        const float sj = s_score[j];
        rank += (sj > sm || (sj == sm && s_tok[j] < tm)) ? 1 : 0;
      }
      int k = k_cur;
      if (rank < n)
        k = k_cur + a.delta_cur;
      else if (rank >= nj - n)
        k = k_cur - a.delta_cur;
      k = clip(k, a.k_min, a.k_max);
      k_out[tm] = k;
      my_sum += static_cast<unsigned long long>(k);
    }
  }
  if (a.role_shuffle) {
    // Role shuffle: token i takes the count of the sequence's r_i-th
    // position, r_i the rank of (key_i, i); a permutation, so my_sum holds.
    // The ranks come from a bitonic sort of the words key << 32 | offset.
    const int len = hi - lo;
    if (len > kMaxJ) {
      if (threadIdx.x == 0) atomicOr(&s_err, kErrCapacity);
    } else {
      constexpr int kPer = kMaxJ / kThreads;
      int n2 = 1;
      while (n2 < len) n2 <<= 1;
      __syncthreads();  // every count of the sequence written, s_raw free
      for (int m = threadIdx.x; m < n2; m += kThreads)
        s_raw[m] = m < len ? (static_cast<uint64_t>(shuffle_key(a.shuffle_seed, lo + m)) << 32) |
                                 static_cast<uint32_t>(m)
                           : ~0ull;  // padding sorts last
      __syncthreads();
      for (int size = 2; size <= n2; size <<= 1) {
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
          for (int m = threadIdx.x; m < n2; m += kThreads) {
            const int o = m ^ stride;
            if (o > m) {
              const uint64_t x = s_raw[m], y = s_raw[o];
              const bool up = (m & size) == 0;
              if ((x > y) == up) {
                s_raw[m] = y;
                s_raw[o] = x;
              }
            }
          }
          __syncthreads();
        }
      }
      int take[kPer], dest[kPer];
#pragma unroll
      for (int u = 0; u < kPer; ++u) {
        const int r = threadIdx.x + u * kThreads;
        dest[u] = -1;
        if (r < len) {
          take[u] = k_out[lo + r];  // count of place r goes to the r-th smallest key
          dest[u] = lo + static_cast<int>(s_raw[r] & 0xffffffffu);
        }
      }
      __syncthreads();  // all old counts read before any is replaced
#pragma unroll
      for (int u = 0; u < kPer; ++u)
        if (dest[u] >= 0) k_out[dest[u]] = take[u];
    }
  }
  // warp sums, then one shared atomic per warp; one store or atomic per CTA
  for (int o = 16; o > 0; o >>= 1) my_sum += __shfl_xor_sync(0xffffffffu, my_sum, o);
  if ((threadIdx.x & 31) == 0) atomicAdd(&s_sum, my_sum);
  __syncthreads();
  if (threadIdx.x == 0) {
    if (sole) {
      if (err) *err = s_err;
      if (k_sum) *k_sum = s_sum;
    } else {
      if (err && s_err) atomicOr(err, s_err);
      if (k_sum) atomicAdd(k_sum, s_sum);
    }
  }
}

// defer = 0: waits for the previous kernel before reading anything.
// defer = 1: launched right behind a kernel that writes none of its inputs
// (the router scores of the same forward); it runs alongside that kernel and
// waits for it only before exiting, so that its own completion still implies
// the completion of everything before it in the stream.
__global__ void __launch_bounds__(kThreads)
    budget_kernel(const float* __restrict__ conf1, const float* __restrict__ conf2,
                  const uint8_t* __restrict__ hist_len, const uint8_t* __restrict__ masked,
                  const int32_t* __restrict__ block_id, const int32_t* __restrict__ seq_off,
                  const int32_t* __restrict__ active_block, int T, AllocArgs a,
                  int32_t* __restrict__ k_out, unsigned long long* __restrict__ k_sum,
                  uint32_t* __restrict__ err, int defer) {
  if (!defer) grid_dep_wait();
  grid_dep_launch();
  budget_body(conf1, conf2, hist_len, masked, block_id, seq_off, active_block, T, a, k_out,
              k_sum, err);
  if (defer) grid_dep_wait();
}

__global__ void wait_selftest_kernel(uint32_t* err, uint64_t limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
  }
  __syncthreads();
  // nobody arrives: the wait must give up after limit_ns and report it
  if (threadIdx.x == 0) {
    if (!mbar_wait(&bar, 0, nullptr, limit_ns)) set_err(err, kErrTimeout);
  }
  __syncthreads();
}

}  // namespace

cudaError_t launch_budget(const float* conf1, const float* conf2,
                          const uint8_t* hist_len, const uint8_t* masked,
                          const int32_t* block_id, const int32_t* seq_off,
                          const int32_t* active_block, int T, int B,
                          const AllocArgs& a, int32_t* k_out,
                          unsigned long long* k_sum, uint32_t* err,
                          cudaStream_t stream, bool alongside) {
  if (B <= 0) return cudaSuccess;
  // programmatic launch when nothing is cleared right before it: a single
  // sequence, or alongside the router scores (the caller cleared first)
  if (B == 1 || alongside)
    return launch_pdl(budget_kernel, dim3(B), dim3(kThreads), 0, stream, conf1, conf2,
                      hist_len, masked, block_id, seq_off, active_block, T, a, k_out,
                      k_sum, err, alongside ? 1 : 0);
  budget_kernel<<<B, kThreads, 0, stream>>>(conf1, conf2, hist_len, masked,
                                            block_id, seq_off, active_block, T, a,
                                            k_out, k_sum, err, 0);
  return cudaGetLastError();
}

cudaError_t launch_wait_selftest(uint32_t* err, uint64_t limit_ns,
                                 cudaStream_t stream) {
  wait_selftest_kernel<<<1, 32, 0, stream>>>(err, limit_ns);
  return cudaGetLastError();
}

}  // namespace rx
