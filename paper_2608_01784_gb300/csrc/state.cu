// state.cu — refinement-state update after one denoising forward of
// block-wise DLM inference (REFLEX Sec. 3.1, Eq. 1), the step that links one
// forward's allocation to the next one's.
//
// Per sequence (one CTA): with a = the active block, J = the masked
// positions of block a and c = the confidences the forward produced,
//   1. commit C = {i in J : c_i >= theta}; when C is empty and J is not, the
//      single most confident member of J (lower position on ties) is
//      committed instead, so that every forward makes progress;
//   2. every position that was masked during the forward records c_i as its
//      newest observation: c^{t-2} <- c^{t-1}, c^{t-1} <- c_i, hist <- min(hist
//      + 1, 2) (the forward predicts every masked position);
//   3. once block a has no masked position left, a advances to a + 1; a
//      sequence whose active index passed its block count Q is finished and
//      left untouched.
#include "common.cuh"
#include "internal.h"

namespace rx {
namespace {

constexpr int kThreads = 1024;

__device__ __forceinline__ uint32_t order_bits(float v) {
  const uint32_t u = __float_as_uint(v);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__global__ void __launch_bounds__(kThreads)
    update_state_kernel(const float* __restrict__ conf_new, float* __restrict__ conf1,
                        float* __restrict__ conf2, uint8_t* __restrict__ hist_len,
                        uint8_t* __restrict__ masked, const int32_t* __restrict__ block_id,
                        const int32_t* __restrict__ seq_off, int32_t* __restrict__ active,
                        const int32_t* __restrict__ num_blocks, int T, float theta,
                        int32_t* __restrict__ committed, uint32_t* __restrict__ err) {
  __shared__ int s_nj, s_nc;
  __shared__ unsigned long long s_best;  // order bits of c << 32 | ~position
  grid_dep_wait();
  grid_dep_launch();
  const int s = blockIdx.x;
  const int lo = seq_off[s], hi = seq_off[s + 1];
  if (lo < 0 || hi > T || lo > hi) {
    if (threadIdx.x == 0) {
      set_err(err, kErrIndex);
      if (committed) committed[s] = 0;
    }
    return;
  }
  const int a = active[s];
  const int q = num_blocks[s];
  if (a < 1 || a > q) {  // finished (a > Q) or invalid (a < 1): unchanged
    if (threadIdx.x == 0) {
      if (a < 1) set_err(err, kErrActive);
      if (committed) committed[s] = 0;
    }
    return;
  }
  if (threadIdx.x == 0) {
    s_nj = 0;
    s_nc = 0;
    s_best = 0ull;
  }
  __syncthreads();
  int my_nj = 0, my_nc = 0;
  unsigned long long my_best = 0ull;
  for (int i = lo + threadIdx.x; i < hi; i += kThreads) {
    if (!masked[i]) continue;
    const float c = conf_new[i];
    if (block_id[i] == a) {
      ++my_nj;
      const float cz = c == 0.0f ? 0.0f : c;  // -0 and +0 are equal confidences
      const unsigned long long key =
          (static_cast<unsigned long long>(order_bits(cz)) << 32) |
          static_cast<unsigned long long>(0xffffffffu - static_cast<uint32_t>(i));
      my_best = key > my_best ? key : my_best;
      if (c >= theta) {
        masked[i] = 0;
        ++my_nc;
      }
    }
    conf2[i] = conf1[i];
    conf1[i] = c;
    const int h = hist_len[i];
    hist_len[i] = static_cast<uint8_t>(h >= 2 ? 2 : h + 1);
  }
  for (int o = 16; o > 0; o >>= 1) {
    my_nj += __shfl_xor_sync(0xffffffffu, my_nj, o);
    my_nc += __shfl_xor_sync(0xffffffffu, my_nc, o);
    const unsigned long long ob = __shfl_xor_sync(0xffffffffu, my_best, o);
    my_best = ob > my_best ? ob : my_best;
  }
  if ((threadIdx.x & 31) == 0) {
    atomicAdd(&s_nj, my_nj);
    atomicAdd(&s_nc, my_nc);
    atomicMax(&s_best, my_best);
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int nc = s_nc;
    if (s_nj > 0 && nc == 0) {  // nothing reached theta: commit the most confident
      const int i = static_cast<int>(0xffffffffu - static_cast<uint32_t>(s_best & 0xffffffffull));
      if (i >= lo && i < hi) {
        masked[i] = 0;
        nc = 1;
      } else {
        set_err(err, kErrIndex);
      }
    }
    if (s_nj - nc == 0) active[s] = a + 1;  // block resolved: advance
    if (committed) committed[s] = nc;
  }
}

}  // namespace

cudaError_t launch_update_state(const float* conf_new, float* conf1, float* conf2,
                                uint8_t* hist_len, uint8_t* masked, const int32_t* block_id,
                                const int32_t* seq_off, int32_t* active,
                                const int32_t* num_blocks, int T, int B, float theta,
                                int32_t* committed, uint32_t* err, cudaStream_t stream) {
  if (B <= 0) return cudaSuccess;
  return launch_pdl(update_state_kernel, dim3(B), dim3(kThreads), 0, stream, conf_new, conf1,
                    conf2, hist_len, masked, block_id, seq_off, active, num_blocks, T, theta,
                    committed, err);
}

}  // namespace rx
