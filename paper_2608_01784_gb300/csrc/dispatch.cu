// dispatch.cu — deterministic token-expert pair compaction for the sparse
// execution of Eq. 2 (REFLEX Sec. 3.2): the pairs (t, j), j < k_t, are laid
// out grouped by expert and, within an expert, in token order, so that each
// expert's rows form one contiguous range of a grouped GEMM.
//
// Three launches, no atomics whose order matters:
//   count   per block of 256 tokens, a bitmask per expert in shared memory
//           (bit = token of the block selected the expert; a token selects
//           an expert at most once) and its popcount per expert;
//   scan    per expert, exclusive prefix over blocks; per-expert totals;
//           exclusive prefix over experts = offsets, and over the 128- and
//           256-row tile counts = tile prefixes for the grouped GEMMs;
//   gather  the row of pair (t, j) is offsets[e] + block prefix + popcount
//           of the lower tokens' bits in the block's masks (kept in global
//           memory by count); X rows are copied into pair order on the way
//           (with REFLEX_FLAG_GATHER_IN_GEMM the CTA-pair GEMM fetches them).
// Short batches whose masks fit in one CTA's shared memory take two: count
// and scan in one CTA, then the gather.
#include "common.cuh"
#include "internal.h"

namespace rx {
namespace {


__device__ __forceinline__ int clamp_k(int kt, int kcap) {
  return kt < 1 ? 1 : (kt > kcap ? kcap : kt);
}

// BLK tokens per block (one CTA of BLK threads), BLK / 32 mask words per
// expert: 32-token blocks up to 4096 tokens (more CTAs for short batches),
// 256-token blocks beyond (fewer blocks for the scan).
template <int BLK>
__device__ void build_masks(uint32_t* mask, const int32_t* ids,
                            const int32_t* k, int T, int E, int k_max,
                            uint32_t* err) {
  constexpr int kBlk = BLK, kWords = BLK / 32;
  for (int i = threadIdx.x; i < E * kWords; i += kBlk) mask[i] = 0u;
  __syncthreads();
  const int t = blockIdx.x * kBlk + threadIdx.x;
  if (t < T) {
    const int kt = clamp_k(k[t], k_max < E ? k_max : E);
    for (int j = 0; j < kt; ++j) {
      const int e = ids[static_cast<int64_t>(t) * k_max + j];
      if (e >= 0 && e < E)
        atomicOr(&mask[e * kWords + (threadIdx.x >> 5)], 1u << (threadIdx.x & 31));
      else
        set_err(err, kErrIndex);
    }
  }
  __syncthreads();
}

template <int BLK>
__global__ void __launch_bounds__(BLK)
    count_kernel(const int32_t* __restrict__ ids, const int32_t* __restrict__ k,
                 int T, int E, int k_max, int32_t* __restrict__ blk_count,
                 uint32_t* __restrict__ blk_mask, uint32_t* __restrict__ err) {
  constexpr int kBlk = BLK, kWords = BLK / 32;
  extern __shared__ uint32_t mask[];
  grid_dep_wait();
  grid_dep_launch();
  build_masks<BLK>(mask, ids, k, T, E, k_max, err);
  uint32_t* gm = blk_mask + static_cast<int64_t>(blockIdx.x) * E * kWords;
  for (int i = threadIdx.x; i < E * kWords; i += kBlk) gm[i] = mask[i];
  for (int e = threadIdx.x; e < E; e += kBlk) {
    int c = 0;
#pragma unroll
    for (int w = 0; w < kWords; ++w) c += __popc(mask[e * kWords + w]);
    blk_count[static_cast<int64_t>(blockIdx.x) * E + e] = c;
  }
}

// Exclusive scan of one value per thread over a block of 1024 threads.
// Exclusive scans of three values per thread over a block of 1024 threads
// (one pass: two block barriers for all three).
struct Scan3 {
  int a, b, c;
};
__device__ Scan3 block_exclusive_scan3(Scan3 v, int (*s_warp)[32], Scan3* total) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  Scan3 x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int ya = __shfl_up_sync(0xffffffffu, x.a, o);
    const int yb = __shfl_up_sync(0xffffffffu, x.b, o);
    const int yc = __shfl_up_sync(0xffffffffu, x.c, o);
    if (lane >= o) {
      x.a += ya;
      x.b += yb;
      x.c += yc;
    }
  }
  if (lane == 31) {
    s_warp[0][wid] = x.a;
    s_warp[1][wid] = x.b;
    s_warp[2][wid] = x.c;
  }
  __syncthreads();
  if (wid < 3) {
    int s = s_warp[wid][lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, s, o);
      if (lane >= o) s += y;
    }
    s_warp[wid][lane] = s;  // inclusive prefix of warp totals
  }
  __syncthreads();
  Scan3 r;
  r.a = (wid > 0 ? s_warp[0][wid - 1] : 0) + x.a - v.a;
  r.b = (wid > 0 ? s_warp[1][wid - 1] : 0) + x.b - v.b;
  r.c = (wid > 0 ? s_warp[2][wid - 1] : 0) + x.c - v.c;
  total->a = s_warp[0][31];
  total->b = s_warp[1][31];
  total->c = s_warp[2][31];
  return r;
}

__global__ void __launch_bounds__(1024)
    scan_kernel(const int32_t* __restrict__ blk_count, int nblk, int E,
                int32_t* __restrict__ blk_off, int32_t* __restrict__ counts,
                int32_t* __restrict__ offsets, int32_t* __restrict__ mt_prefix,
                int32_t* __restrict__ mt2_prefix, int32_t* __restrict__ totals) {
  __shared__ int s_warp3[3][32];
  __shared__ int s_total[1024];
  grid_dep_wait();
  grid_dep_launch();
  // G threads per expert (a power of two, at most 32, G * E <= 1024): thread
  // (e, g) loads its chunk of the expert's block counts in one go (one L2
  // round trip instead of one per eight blocks), a segmented warp scan gives
  // the chunks' prefixes, and each thread writes its blocks' offsets
  int G = 1;
  while (G < 32 && 2 * G * E <= 1024) G *= 2;
  const int chunk = (nblk + G - 1) / G;
  {
    const int e = threadIdx.x / G, g = threadIdx.x % G;
    const int b_lo = min(nblk, g * chunk), b_hi = min(nblk, b_lo + chunk);
    int local = 0;
    if (e < E) {
#pragma unroll 8
      for (int b = b_lo; b < b_hi; ++b) local += blk_count[static_cast<int64_t>(b) * E + e];
    }
    int incl = local;  // inclusive prefix over the group's lanes (width G)
    for (int o = 1; o < G; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, o, G);
      if (g >= o) incl += v;
    }
    if (e < E) {
      int run = incl - local;
#pragma unroll 8
      for (int b = b_lo; b < b_hi; ++b) {
        const int64_t idx = static_cast<int64_t>(b) * E + e;
        const int c = blk_count[idx];
        blk_off[idx] = run;
        run += c;
      }
      if (g == G - 1) s_total[e] = incl;
    }
  }
  __syncthreads();
  const int e = threadIdx.x;  // E <= 1024
  const int run = e < E ? s_total[e] : 0;
  if (e < E) counts[e] = run;
  // pairs, 128-row tiles and 256-row tiles (CTA-pair GEMM) per expert
  Scan3 tot;
  const Scan3 pre = block_exclusive_scan3(
      Scan3{e < E ? run : 0, e < E ? (run + kTileM - 1) / kTileM : 0,
            e < E ? (run + 2 * kTileM - 1) / (2 * kTileM) : 0},
      s_warp3, &tot);
  const int off = pre.a, toff = pre.b, toff2 = pre.c;
  const int total_pairs = tot.a, total_tiles = tot.b, total_tiles2 = tot.c;
  if (e < E) {
    offsets[e] = off;
    mt_prefix[e] = toff;
    mt2_prefix[e] = toff2;
  }
  if (e == 0) {
    offsets[E] = total_pairs;
    mt_prefix[E] = total_tiles;
    mt2_prefix[E] = total_tiles2;
    totals[0] = total_pairs;
    totals[1] = total_tiles;
    totals[2] = total_tiles2;
  }
}

// Short batches: the count and scan steps in one CTA.  Every pair sets its
// token's bit in the (32-token block, expert) mask word in shared memory
// (a token selects an expert at most once; OR is order-free); then, per
// expert, the block prefixes of the popcounts and the total, and the expert
// and tile prefixes as in scan_kernel.  The masks and block prefixes go to
// global memory for gather_scatter_kernel.
__global__ void __launch_bounds__(1024)
    count_scan_kernel(const int32_t* __restrict__ ids, const int32_t* __restrict__ k,
                      int T, int E, int k_max, int nblk, int32_t* __restrict__ blk_off,
                      int32_t* __restrict__ counts, int32_t* __restrict__ offsets,
                      int32_t* __restrict__ mt_prefix, int32_t* __restrict__ mt2_prefix,
                      int32_t* __restrict__ totals, uint32_t* __restrict__ blk_mask,
                      uint32_t* __restrict__ err) {
  extern __shared__ uint32_t s_mask[];  // [nblk][E]: bit = token of the block
  __shared__ int s_warp3[3][32];
  grid_dep_wait();
  grid_dep_launch();
  for (int i = threadIdx.x; i < nblk * E; i += 1024) s_mask[i] = 0u;
  __syncthreads();
  const int kcap = k_max < E ? k_max : E;
  for (int t = threadIdx.x; t < T; t += 1024) {
    const int kt = clamp_k(k[t], kcap);
    uint32_t* row = s_mask + (t / kDispatchBlockSmall) * E;
    const uint32_t bit = 1u << (t % kDispatchBlockSmall);
    for (int j = 0; j < kt; ++j) {
      const int e = ids[static_cast<int64_t>(t) * k_max + j];
      if (e >= 0 && e < E)
        atomicOr(&row[e], bit);
      else
        set_err(err, kErrIndex);
    }
  }
  __syncthreads();
  const int e = threadIdx.x;  // E <= 1024
  int run = 0;
  if (e < E) {
    for (int b = 0; b < nblk; ++b) {
      const int64_t i = static_cast<int64_t>(b) * E + e;
      const uint32_t m = s_mask[b * E + e];
      blk_off[i] = run;
      blk_mask[i] = m;
      run += __popc(m);
    }
    counts[e] = run;
  }
  Scan3 tot;
  const Scan3 pre = block_exclusive_scan3(
      Scan3{e < E ? run : 0, e < E ? (run + kTileM - 1) / kTileM : 0,
            e < E ? (run + 2 * kTileM - 1) / (2 * kTileM) : 0},
      s_warp3, &tot);
  const int off = pre.a, toff = pre.b, toff2 = pre.c;
  const int total_pairs = tot.a, total_tiles = tot.b, total_tiles2 = tot.c;
  if (e < E) {
    offsets[e] = off;
    mt_prefix[e] = toff;
    mt2_prefix[e] = toff2;
  }
  if (e == 0) {
    offsets[E] = total_pairs;
    mt_prefix[E] = total_tiles;
    mt2_prefix[E] = total_tiles2;
    totals[0] = total_pairs;
    totals[1] = total_tiles;
    totals[2] = total_tiles2;
  }
}

// Token-order gather with the scatter step (xp == nullptr: the pairs are
// placed and no row is copied; the grouped GEMM gathers the rows itself).  W warps per token (W = 1 for
// long batches), each reading one 1/W segment of the token's hidden row
// once (up to 8 16-byte vectors per lane in flight) and writing it to each
// of the token's k_t pair rows, so every hidden row crosses HBM once however
// many experts selected it; short batches split rows across warps so that
// every SM gets work.  Lane j of a warp of token t places pair (t, j) at
// offsets[e] + block prefix + the popcount of the lower tokens' bits in its
// block's KW mask words of expert e (the pairs of expert e in token order);
// the warp of the row's first segment writes perm and row_of.
template <typename Te, int KW>
__global__ void __launch_bounds__(256)
    gather_scatter_kernel(const Te* __restrict__ x, const int32_t* __restrict__ ids,
                          const int32_t* __restrict__ k, const uint32_t* __restrict__ blk_mask,
                          const int32_t* __restrict__ blk_off,
                          const int32_t* __restrict__ offsets, int E, int k_max, int cap_rows,
                          int T, int d, int wpt, int32_t* __restrict__ perm,
                          int32_t* __restrict__ row_of, Te* __restrict__ xp,
                          uint32_t* __restrict__ err) {
  constexpr int kVecElems = 16 / sizeof(Te);
  constexpr int kMaxVec = 8;
  grid_dep_wait();
  grid_dep_launch();
  const int lane = threadIdx.x & 31;
  const int warps = gridDim.x * 8;
  const int row_vecs = d / kVecElems;
  const int seg_vecs = row_vecs / wpt;
  const int units = T * wpt;
  const int kcap = k_max < E ? k_max : E;
  for (int u = blockIdx.x * 8 + (threadIdx.x >> 5); u < units; u += warps) {
    const int t = u / wpt;
    const int seg = u % wpt;
    const int v0 = seg * seg_vecs;
    const int kt = clamp_k(k[t], kcap);
    // the row segment's first vectors do not depend on the pair rows: their
    // loads overlap the position lookups
    const uint4* src = reinterpret_cast<const uint4*>(x + static_cast<int64_t>(t) * d) + v0;
    uint4 v[kMaxVec];
    if (xp != nullptr) {
#pragma unroll
      for (int i = 0; i < kMaxVec; ++i) {
        const int q = lane + 32 * i;
        if (q < seg_vecs) v[i] = __ldg(src + q);
      }
    }
    int my_row = -1;
    if (lane < k_max) {
      const int64_t o = static_cast<int64_t>(t) * k_max + lane;
      if (lane < kt) {
        const int e = ids[o];
        if (e >= 0 && e < E) {
          const int tb = t % (32 * KW);  // token within its block
          const int64_t bi = static_cast<int64_t>(t / (32 * KW)) * E + e;
          const uint32_t below = (1u << (tb & 31)) - 1u;
          int local;
          if constexpr (KW == 1) {
            local = __popc(blk_mask[bi] & below);
          } else {
            static_assert(KW == 8, "32- or 256-token blocks");
            const uint4* mv = reinterpret_cast<const uint4*>(blk_mask + bi * KW);
            const uint4 m0 = mv[0], m1 = mv[1];
            const uint32_t m[8] = {m0.x, m0.y, m0.z, m0.w, m1.x, m1.y, m1.z, m1.w};
            const int w = tb >> 5;
            local = 0;
#pragma unroll
            for (int i = 0; i < 8; ++i)
              local += i < w ? __popc(m[i]) : (i == w ? __popc(m[i] & below) : 0);
          }
          my_row = offsets[e] + blk_off[bi] + local;
          if (my_row < 0 || my_row >= cap_rows) {
            set_err(err, kErrIndex);
            my_row = -1;
          }
        }
      }
      if (seg == 0) {
        row_of[o] = my_row;
        if (my_row >= 0) perm[my_row] = static_cast<int32_t>(o);
      }
    }
    if (xp == nullptr) continue;  // placement only
    for (int base = 0; base < seg_vecs; base += 32 * kMaxVec) {
      if (base > 0) {
#pragma unroll
        for (int i = 0; i < kMaxVec; ++i) {
          const int q = base + lane + 32 * i;
          if (q < seg_vecs) v[i] = __ldg(src + q);
        }
      }
      for (int j = 0; j < kt; ++j) {
        const int r = __shfl_sync(0xffffffffu, my_row, j);
        if (r < 0) continue;
        uint4* dst = reinterpret_cast<uint4*>(xp + static_cast<int64_t>(r) * d) + v0;
#pragma unroll
        for (int i = 0; i < kMaxVec; ++i) {
          const int q = base + lane + 32 * i;
          if (q < seg_vecs) dst[q] = v[i];
        }
      }
    }
  }
}

// warps per token for the gather (enough warps for 16 per SM, each segment
// whole 16-byte vectors) and the grid
void gather_shape(int dtype, int T, int d, int num_sms, bool copy, int* wpt_out,
                  int* grid_out) {
  const int row_vecs = d * (dtype == 0 ? 4 : 2) / 16;
  int wpt = 1;
  while (copy && wpt < 8 && static_cast<int64_t>(T) * wpt < 16LL * num_sms &&
         row_vecs % (2 * wpt) == 0)
    wpt *= 2;
  const int64_t warps = static_cast<int64_t>(T) * wpt;
  int grid = static_cast<int>((warps + 7) / 8);
  if (grid > 16 * num_sms) grid = 16 * num_sms;
  *wpt_out = wpt;
  *grid_out = grid;
}

}  // namespace

// count and scan over BLK-token blocks (the gather places the pairs)
template <int BLK>
cudaError_t launch_dispatch_blk(const int32_t* ids, const int32_t* k, int T, int E, int k_max,
                                const DispatchBufs& b, cudaStream_t stream) {
  const int nblk = (T + BLK - 1) / BLK;
  const size_t smem = static_cast<size_t>(E) * (BLK / 32) * sizeof(uint32_t);
  if (smem > 48 * 1024) {
    const cudaError_t e1 = cudaFuncSetAttribute(
        count_kernel<BLK>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e1 != cudaSuccess) return e1;
  }
  cudaError_t e = launch_pdl(count_kernel<BLK>, dim3(nblk), dim3(BLK), smem, stream, ids, k, T,
                             E, k_max, b.blk_count, b.blk_mask, b.err);
  if (e != cudaSuccess) return e;
  return launch_pdl(scan_kernel, dim3(1), dim3(1024), 0, stream, b.blk_count, nblk, E,
                    b.blk_off, b.counts, b.offsets, b.mt_prefix, b.mt2_prefix, b.totals);
}

// Short batches whose block masks fit in shared memory: count + scan in one
// CTA.
constexpr size_t kCountScanSmem = 160 * 1024;

static cudaError_t launch_count_scan(const int32_t* ids, const int32_t* k, int T, int E,
                                    int k_max, const DispatchBufs& b, cudaStream_t stream) {
  const int nblk = (T + kDispatchBlockSmall - 1) / kDispatchBlockSmall;
  const size_t cs_smem = static_cast<size_t>(nblk) * E * sizeof(uint32_t);
  if (cs_smem > 48 * 1024) {
    const cudaError_t e = cudaFuncSetAttribute(
        count_scan_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)cs_smem);
    if (e != cudaSuccess) return e;
  }
  return launch_pdl(count_scan_kernel, dim3(1), dim3(1024), cs_smem, stream, ids, k, T, E,
                    k_max, nblk, b.blk_off, b.counts, b.offsets, b.mt_prefix, b.mt2_prefix,
                    b.totals, b.blk_mask, b.err);
}

template <typename Te, int KW>
static cudaError_t launch_gather_scatter(const Te* hidden, const int32_t* ids, const int32_t* k,
                                         int T, int E, int k_max, int cap_rows, int d,
                                         const DispatchBufs& b, Te* x_perm, int num_sms,
                                         cudaStream_t stream) {
  int wpt, grid;
  gather_shape(sizeof(Te) == 4 ? 0 : 1, T, d, num_sms, x_perm != nullptr, &wpt, &grid);
  return launch_pdl(gather_scatter_kernel<Te, KW>, dim3(grid), dim3(256), 0, stream, hidden,
                    ids, k, static_cast<const uint32_t*>(b.blk_mask),
                    static_cast<const int32_t*>(b.blk_off), static_cast<const int32_t*>(b.offsets),
                    E, k_max, cap_rows, T, d, wpt, b.perm, b.row_of, x_perm, b.err);
}

template <typename Te>
static cudaError_t dispatch_gather(const Te* hidden, const int32_t* ids, const int32_t* k,
                                   int T, int E, int k_max, int cap_rows, int d,
                                   const DispatchBufs& b, Te* x_perm, int num_sms,
                                   cudaStream_t stream) {
  if (T == 0) return cudaSuccess;
  cudaError_t e;
  if (dispatch_block(T) == kDispatchBlockSmall) {
    e = static_cast<size_t>((T + kDispatchBlockSmall - 1) / kDispatchBlockSmall) * E *
                    sizeof(uint32_t) <= kCountScanSmem
            ? launch_count_scan(ids, k, T, E, k_max, b, stream)
            : launch_dispatch_blk<kDispatchBlockSmall>(ids, k, T, E, k_max, b, stream);
    if (e != cudaSuccess) return e;
    return launch_gather_scatter<Te, 1>(hidden, ids, k, T, E, k_max, cap_rows, d, b, x_perm,
                                        num_sms, stream);
  }
  e = launch_dispatch_blk<kDispatchBlock>(ids, k, T, E, k_max, b, stream);
  if (e != cudaSuccess) return e;
  return launch_gather_scatter<Te, kDispatchBlock / 32>(hidden, ids, k, T, E, k_max, cap_rows,
                                                        d, b, x_perm, num_sms, stream);
}

cudaError_t launch_dispatch_gather(int dtype, const void* hidden, const int32_t* ids,
                                   const int32_t* k, int T, int E, int k_max, int cap_rows,
                                   int d, const DispatchBufs& b, void* x_perm, int num_sms,
                                   cudaStream_t stream) {
  if (dtype == 0)
    return dispatch_gather(static_cast<const float*>(hidden), ids, k, T, E, k_max, cap_rows, d,
                           b, static_cast<float*>(x_perm), num_sms, stream);
  return dispatch_gather(static_cast<const __nv_bfloat16*>(hidden), ids, k, T, E, k_max,
                         cap_rows, d, b, static_cast<__nv_bfloat16*>(x_perm), num_sms, stream);
}

}  // namespace rx
