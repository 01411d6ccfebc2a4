// experts_tc.cu — grouped SwiGLU expert GEMMs over ragged per-expert row
// ranges on the 5th-generation tensor cores (tcgen05.mma, accumulators in
// TMEM, operands staged by TMA), for the sparse execution of Eq. 2 (REFLEX
// Sec. 3.2).  Routed-expert work is 6 * d * inter FLOPs per selected pair
// (Eq. 10), two thirds in the gate/up GEMM and one third in the down GEMM.
//
// Problem.  Rows of the pair-ordered input A are grouped by expert
// (rows [offsets[e], offsets[e+1]) belong to expert e).  For each group:
//   SwiGLU mode: out[r, c] = silu(A_r . Wg[e, c]) * (A_r . Wu[e, c])
//   Down mode:   out[r, n] = A_r . Wd[e, n]
// with every operand K-major bf16 and fp32 accumulation; out is bf16.
//
// Tiles.  An output tile is 128 rows (one m-tile of a group; rows past the
// group's end are computed from the next rows or TMA zero fill and never
// stored) by BN columns.  In SwiGLU mode the BN-row weight tile is the
// BN/2 gate rows followed by the matching BN/2 up rows, loaded by two TMA
// boxes, so one MMA chain yields gate and up side by side in TMEM and the
// epilogue emits BN/2 activations.  Tiles are numbered expert-major, then
// n-tile, then m-tile, so CTAs running at the same time share weight tiles
// in L2.
//
// Kernel.  Persistent: one CTA per SM walks tiles blockIdx.x, +gridDim.x, ...
//   warp 0     TMA producer: 192 KB ring of (A 128x64, B BNx64) bf16 stages
//              (4 for BN 256, 6 for 128, 8 for 64), 128-byte swizzle,
//              completion on a per-stage mbarrier;
//   warp 1     allocates 2*BN TMEM columns (two accumulators) and issues
//              tcgen05.mma (M=128, N=BN, K=16) from one thread; each stage
//              is released with tcgen05.commit when its MMAs have read it;
//   warps 2-5  epilogue: tcgen05.ld 32x32b of their TMEM lane quarter,
//              SwiGLU or conversion, 16-byte stores; the accumulator is
//              handed back through an mbarrier, so the epilogue of tile i
//              overlaps the main loop of tile i+1.
// A tile number maps to (expert, n-tile, rows) through the per-expert tile
// prefix, copied into shared memory once per CTA (TileIndex).  Every wait is
// bounded (2 s); on expiry the CTA records the timeout in the error word,
// drains its outstanding TMA loads and MMAs, frees TMEM and exits.  The
// 2-SM (CTA pair) variant further down has its own description.
#include "common.cuh"
#include "internal.h"

namespace rx {
namespace {

constexpr int BM = kTileM;   // 128
constexpr int BK = 64;       // 64 bf16 = 128 bytes = one swizzle row
constexpr int UMMA_K = 16;
constexpr int kThreads = 192;
// scores mode: four more warps (6-9) that sum the squares of each A row from
// the shared-memory stages while the MMAs read them (token norms for the
// router screen's interval)
constexpr int kThreadsScores = 320;
constexpr int kRingBytes = 192 * 1024;  // TMA ring budget per CTA
constexpr uint64_t kWaitNs = 2000000000ull;
constexpr uint64_t kDrainNs = 1000000000ull;

enum { kModeSwiGLU = 0, kModeDown = 1, kModeScores = 2 };

template <int BN>
struct Cfg {
  static constexpr int kABytes = BM * BK * 2;
  static constexpr int kBBytes = BN * BK * 2;
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kStages = kRingBytes / kStageBytes;  // 4 (BN 256), 6 (BN 128)
  static constexpr int kTmemCols = 2 * BN;
  static constexpr int kBarBytes = 256;
  static constexpr int kIndexInts = 2 * 1025;  // both prefix arrays, E <= 1024
  static constexpr int kSmemBytes = kStages * kStageBytes + kBarBytes + kIndexInts * 4 + 1024;
  static_assert(kStages >= 2 && kStages <= 8, "ring depth");
};

struct KParams {
  int K;
  int n_tiles;           // column tiles per group
  int b_rows_per_group;
  int b_up_offset;
  GroupRows g;
  const int32_t* mt_prefix;  // [E+1] prefix of tile counts (grouped mode)
  int max_mtiles;            // host upper bound of m-tiles
  int tile_rows;             // rows per tile: 128 (1-SM) or 256 (CTA pair)
  __nv_bfloat16* out;
  int ldo;
  uint32_t* err;
  // scores mode (dense, fp32 out): K is cut into k_splits slices; slice ks of
  // tile (m, n) writes out_f32 + ks * split_stride; columns >= n_valid dropped
  int k_splits;
  float* out_f32;
  int64_t split_stride;
  int n_valid;
  // 1: launched right behind a kernel that writes none of this kernel's
  // inputs or outputs; start at once and wait for it only before exiting
  int defer_wait;
  // SwiGLU: map_b is the 3D {K, inter, 2 groups} map of tc_gate_up_3d
  int b3d;
  // scores mode, k_splits == 1: sum of squares of every A row (fp32), nullable
  float* norm_out;
  // CTA pairs: whole 32-row output chunks leave by TMA store (map_out)
  int tma_out;
  // SwiGLU on CTA pairs: A rows gathered from the token rows (TcGemmArgs)
  const int32_t* gather_perm;
  int gather_kmax;
  int gather_tokens;
};

// ---- PTX wrappers ---------------------------------------------------------
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive1(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map,
                                            int c0, int c1, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(bar)
      : "memory");
}
// L2 eviction priority for TMA loads.  A weight tile of a group that fits in
// one m-tile is read by exactly one CTA, so it is loaded evict-first and the
// weight stream does not push the group rows, activations and outputs out of
// L2 (LLaDA-MoE layer: gate/up GEMM 102 -> 97 us).  Every other load is a
// plain load: evict-first on weights that several m-tiles read makes the
// second reader miss, and an explicit evict-normal hint measured slower than
// no hint (2-5% at 4096-16384 tokens).
constexpr int kPolFirst = 0;
__device__ __forceinline__ uint64_t l2_policy(int) {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}
__device__ __forceinline__ void tma_load_2d_hint(uint32_t dst, const CUtensorMap* map, int c0,
                                                 int c1, uint32_t bar, uint64_t pol) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      ".L2::cache_hint [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(bar), "l"(pol)
      : "memory");
}
// 3D boxes: the gate and up blocks of one weight tile in one copy (the map's
// dims are {K, rows per half, halves}: halves 2e and 2e + 1 of expert e)
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, int c0,
                                            int c1, int c2, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(bar)
      : "memory");
}
__device__ __forceinline__ void tma_load_3d_hint(uint32_t dst, const CUtensorMap* map, int c0,
                                                 int c1, int c2, uint32_t bar, uint64_t pol) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      ".L2::cache_hint [%0], [%1, {%2, %3, %4}], [%5], %6;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(bar), "l"(pol)
      : "memory");
}
__device__ __forceinline__ void prefetch_map(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map))
               : "memory");
}
// Shared-memory matrix descriptor: K-major tile with 128-byte swizzle, rows
// of 128 bytes, 8-row groups 1024 bytes apart.
__device__ __forceinline__ uint64_t desc_sw128(uint32_t saddr) {
  uint64_t desc = static_cast<uint64_t>((saddr >> 4) & 0x3FFFu);  // start
  desc |= static_cast<uint64_t>(1) << 16;            // leading offset (unused)
  desc |= static_cast<uint64_t>(1024 >> 4) << 32;    // stride offset
  desc |= static_cast<uint64_t>(1) << 46;            // descriptor version
  desc |= static_cast<uint64_t>(2) << 61;            // 128-byte swizzle
  return desc;
}
// Instruction descriptor of kind::f16: bf16 A and B, fp32 accumulator,
// both K-major, M = 128, N = n.
__host__ __device__ constexpr uint32_t idesc_bf16(int n) {
  return (1u << 4) | (1u << 7) | (1u << 10) |
         (static_cast<uint32_t>(n >> 3) << 17) |
         (static_cast<uint32_t>(BM >> 4) << 24);
}
__device__ __forceinline__ void mma_bf16(uint32_t tmem_d, uint64_t da,
                                         uint64_t db, uint32_t idesc,
                                         uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(tmem_d),
      "l"(da), "l"(db), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void mma_commit(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
      : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tmem_alloc(uint32_t slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(slot),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr),
               "r"(ncols)
               : "memory");
}
// 32 TMEM lanes x 32 consecutive fp32 columns: one column per register.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, "
      "[%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]),
        "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]),
        "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]),
        "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
        "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]),
        "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld_wait() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// ---- tile numbering -------------------------------------------------------
struct Tile {
  int e, n, row0, rows;
  int mtiles;  // m-tiles of the tile's group (readers of each weight tile)
  int ks;      // K slice (scores mode; 0 otherwise)
};

// The group prefix arrays a tile lookup reads: copies in shared memory where
// they fit, else the global arrays.  Looking a tile up takes a binary search
// over the experts; from global memory that is a chain of about log2(E) + 2
// dependent L2 loads (about 3 us), longer than the ring's lead over the MMAs
// at each tile start, so the copies are made once per CTA.
struct TileIndex {
  const int32_t* pref;  // [E+1] tile-count prefix (p.mt_prefix)
  const int32_t* offs;  // [E+1] row offsets (p.g.offsets)
};
// Every thread of the CTA calls this (it synchronises the CTA) after the
// kernel's dependency wait; cache holds cap ints.
__device__ __forceinline__ TileIndex load_tile_index(const KParams& p, int32_t* cache,
                                                     int cap) {
  TileIndex ix{p.mt_prefix, p.g.offsets};
  if (p.g.offsets == nullptr) return ix;
  const int n = p.g.E + 1;
  const bool both = 2 * n <= cap, pref_only = !both && n <= cap;
  if (both || pref_only) {
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
      cache[i] = p.mt_prefix[i];
      if (both) cache[n + i] = p.g.offsets[i];
    }
    __syncthreads();
    ix.pref = cache;
    if (both) ix.offs = cache + n;
  }
  return ix;
}

__device__ __forceinline__ int total_tiles(const KParams& p, const TileIndex& ix) {
  int mt;
  if (p.g.offsets == nullptr) {
    mt = (p.g.dense_rows + p.tile_rows - 1) / p.tile_rows * p.k_splits;
  } else {
    mt = ix.pref[p.g.E];
    if (mt < 0) mt = 0;
    if (mt > p.max_mtiles) mt = p.max_mtiles;
  }
  return mt * p.n_tiles;
}

// Tile t -> (expert, n-tile, rows); false when the workspace is inconsistent.
__device__ __forceinline__ bool decode_tile(const KParams& p, const TileIndex& ix, int t,
                                            Tile& o) {
  if (p.g.offsets == nullptr) {
    const int mt = (p.g.dense_rows + p.tile_rows - 1) / p.tile_rows;
    const int per = mt * p.n_tiles;
    o.ks = t / per;
    t -= o.ks * per;
    o.e = 0;
    o.n = t / mt;
    o.row0 = (t % mt) * p.tile_rows;
    o.rows = min(p.tile_rows, p.g.dense_rows - o.row0);
    o.mtiles = mt;
    return o.ks < p.k_splits;
  }
  o.ks = 0;
  int lo = 0, hi = p.g.E;  // n_tiles*prefix[lo] <= t < n_tiles*prefix[hi]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (p.n_tiles * ix.pref[mid] <= t) lo = mid; else hi = mid;
  }
  const int mt_e = ix.pref[lo + 1] - ix.pref[lo];
  if (mt_e <= 0) return false;
  const int l = t - p.n_tiles * ix.pref[lo];
  o.e = lo;
  o.mtiles = mt_e;
  o.n = l / mt_e;
  o.row0 = ix.offs[lo] + (l % mt_e) * p.tile_rows;
  o.rows = min(p.tile_rows, ix.offs[lo + 1] - o.row0);
  return o.n < p.n_tiles && o.row0 >= 0 && o.rows > 0 &&
         o.row0 + o.rows <= p.g.cap_rows;
}

template <int BN, int MODE>
__global__ void __launch_bounds__(MODE == kModeScores ? kThreadsScores : kThreads, 1)
    grouped_gemm_kernel(const __grid_constant__ CUtensorMap map_a,
                        const __grid_constant__ CUtensorMap map_b,
                        const KParams p) {
  using C = Cfg<BN>;
  constexpr int kStages = C::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* sa = smem;
  uint8_t* sb = smem + kStages * C::kABytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kStages * C::kStageBytes);
  uint64_t* full = bars;
  uint64_t* empty = bars + kStages;
  uint64_t* acc_full = bars + 2 * kStages;
  uint64_t* acc_empty = bars + 2 * kStages + 2;
  uint64_t* drain = bars + 2 * kStages + 4;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * kStages + 5);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  const bool norms = MODE == kModeScores && p.norm_out != nullptr;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], norms ? 5 : 1);  // the MMA commit (+ 4 norm warps)
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], 4);  // one arrival per epilogue warp
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_map(&map_a);
    prefetch_map(&map_b);
  }
  if (warp == 1) tmem_alloc(smem_addr(tmem_slot), C::kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  // the tile count and every operand come from earlier kernels
  if (!p.defer_wait) grid_dep_wait();
  grid_dep_launch();
  const TileIndex ix = load_tile_index(
      p, reinterpret_cast<int32_t*>(smem + kStages * C::kStageBytes + C::kBarBytes),
      C::kIndexInts);
  const int ntiles = total_tiles(p, ix);
  const int nk = p.K / BK / p.k_splits;  // k-blocks per tile

  if (warp == 0 && lane == 0) {
    // ---------------- TMA producer ----------------
    int stage = 0;
    uint32_t phase = 0;
    uint32_t issued_mask = 0, issued_phase = 0;
    bool ok = true;
    const bool grouped = p.g.offsets != nullptr;
    const uint64_t pol_once = l2_policy(kPolFirst);
    for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x) {
      Tile tl;
      if (!decode_tile(p, ix, t, tl)) {
        set_err(p.err, kErrIndex);
        *abort_flag = 1;
        break;
      }
      const bool once = grouped && tl.mtiles == 1;  // one reader per weight tile
      for (int kb = 0; kb < nk; ++kb) {
        if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, kWaitNs)) {
          ok = false;
          break;
        }
        const uint32_t fb = smem_addr(&full[stage]);
        mbar_expect_tx(fb, C::kStageBytes);
        const int k0 = (tl.ks * nk + kb) * BK;
        tma_load_2d(smem_addr(sa + stage * C::kABytes), &map_a, k0, tl.row0, fb);
        const uint32_t b_dst = smem_addr(sb + stage * C::kBBytes);
        const int wr = tl.e * p.b_rows_per_group + tl.n * (MODE == kModeSwiGLU ? BN / 2 : BN);
        auto load_b = [&](uint32_t dst, int row) {
          if (once) tma_load_2d_hint(dst, &map_b, k0, row, fb, pol_once);
          else tma_load_2d(dst, &map_b, k0, row, fb);
        };
        if (MODE == kModeSwiGLU && p.b3d) {
          // gate rows then up rows of the tile, one copy
          if (once) tma_load_3d_hint(b_dst, &map_b, k0, tl.n * (BN / 2), 2 * tl.e, fb, pol_once);
          else tma_load_3d(b_dst, &map_b, k0, tl.n * (BN / 2), 2 * tl.e, fb);
        } else {
          load_b(b_dst, wr);
          if (MODE == kModeSwiGLU) load_b(b_dst + (BN / 2) * BK * 2, wr + p.b_up_offset);
        }
        issued_mask |= 1u << stage;
        issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
        if (++stage == kStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
    if (!ok) {
      set_err(p.err, kErrTimeout);
      *abort_flag = 1;
    }
    if (*abort_flag) {
      // every issued load must land before the CTA may exit
      for (int s = 0; s < kStages; ++s)
        if (issued_mask & (1u << s))
          mbar_wait(&full[s], (issued_phase >> s) & 1u, nullptr, kDrainNs);
    }
  } else if (warp == 1 && lane == 0) {
    // ---------------- MMA issuer ----------------
    constexpr uint32_t idesc = idesc_bf16(BN);
    int stage = 0;
    uint32_t phase = 0;
    int lt = 0;
    bool ok = true, issued_any = false;
    for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x, ++lt) {
      const int ab = lt & 1;
      const uint32_t acc_phase = (lt >> 1) & 1;
      if (!mbar_wait(&acc_empty[ab], acc_phase ^ 1u, abort_flag, kWaitNs)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(ab * BN);
      for (int kb = 0; kb < nk; ++kb) {
        if (!mbar_wait(&full[stage], phase, abort_flag, kWaitNs)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a0 = smem_addr(sa + stage * C::kABytes);
        const uint32_t b0 = smem_addr(sb + stage * C::kBBytes);
#pragma unroll
        for (int k = 0; k < BK / UMMA_K; ++k) {
          mma_bf16(d_tmem, desc_sw128(a0 + k * UMMA_K * 2),
                   desc_sw128(b0 + k * UMMA_K * 2), idesc,
                   (kb > 0 || k > 0) ? 1u : 0u);
        }
        issued_any = true;
        mma_commit(smem_addr(&empty[stage]));
        if (++stage == kStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
      if (!ok) break;
      mma_commit(smem_addr(&acc_full[ab]));
    }
    if (!ok) {
      set_err(p.err, kErrTimeout);
      *abort_flag = 1;
    }
    if (*abort_flag && issued_any) {
      // MMAs in flight must finish before TMEM is freed
      mma_commit(smem_addr(drain));
      mbar_wait(drain, 0, nullptr, kDrainNs);
    }
  } else if (MODE == kModeScores && warp >= 6) {
    // ---------------- row norms (scores mode) ----------------
    // warp 6 + q sums the squares of A rows 32 q .. 32 q + 31 of every tile,
    // one row per lane, reading each stage as the MMAs do and releasing it
    // on the stage's "empty" barrier next to the MMA commit
    if (norms) {
      const int r = (warp - 6) * 32 + lane;
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < ntiles && ok; t += gridDim.x) {
        Tile tl;
        const bool tile_ok = decode_tile(p, ix, t, tl);
        float ss = 0.f;
        for (int kb = 0; kb < nk; ++kb) {
          // every lane observes the stage's completion before reading it
          const bool w = __all_sync(0xffffffffu,
                                    mbar_wait(&full[stage], phase, abort_flag, kWaitNs));
          if (!w) {
            ok = false;
            break;
          }
          // row r of the 128-byte-swizzled A stage: 16-byte chunk c at
          // r * 128 + ((c ^ (r & 7)) << 4)
          const uint8_t* rowp = sa + stage * C::kABytes + r * 128;
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            const uint4 q = *reinterpret_cast<const uint4*>(rowp + ((c ^ (r & 7)) << 4));
            const uint32_t wd[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const float lo = __uint_as_float(wd[i] << 16);
              const float hi = __uint_as_float(wd[i] & 0xffff0000u);
              ss = fmaf(lo, lo, ss);
              ss = fmaf(hi, hi, ss);
            }
          }
          fence_proxy_async_smem();  // the reads above, before the next TMA fill
          __syncwarp();
          if (lane == 0) mbar_arrive1(smem_addr(&empty[stage]));
          if (++stage == kStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (ok && tile_ok && r < tl.rows) p.norm_out[tl.row0 + r] = ss;
      }
      if (!ok && lane == 0) {
        if (!*abort_flag) set_err(p.err, kErrTimeout);
        *abort_flag = 1;
      }
    }
  } else if (warp >= 2) {
    // ---------------- epilogue ----------------
    const int quarter = warp & 3;  // TMEM lanes 32*quarter .. +31
    const int row = quarter * 32 + lane;
    int lt = 0;
    for (int t = blockIdx.x; t < ntiles; t += gridDim.x, ++lt) {
      Tile tl;
      const bool tile_ok = decode_tile(p, ix, t, tl);
      const int ab = lt & 1;
      const uint32_t acc_phase = (lt >> 1) & 1;
      int ok = 1;
      if (lane == 0) ok = mbar_wait(&acc_full[ab], acc_phase, abort_flag, kWaitNs) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) {
        if (lane == 0) {
          if (!*abort_flag) set_err(p.err, kErrTimeout);
          *abort_flag = 1;
        }
        break;
      }
      tc_fence_after();
      const uint32_t tbase = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) +
                             static_cast<uint32_t>(ab * BN);
      const bool store = tile_ok && row < tl.rows;
      __nv_bfloat16* orow =
          p.out + static_cast<int64_t>(tl.row0 + (store ? row : 0)) * p.ldo;
      if (MODE == kModeScores) {
        float* srow = p.out_f32 + tl.ks * p.split_stride +
                      static_cast<int64_t>(tl.row0 + (store ? row : 0)) * p.ldo;
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          uint32_t v32[32];
          tmem_ld32(tbase + c, v32);
          tmem_ld_wait();
          const int col0 = tl.n * BN + c;
          if (store) {
            if (col0 + 32 <= p.n_valid && (p.ldo & 3) == 0) {
              float4* dst = reinterpret_cast<float4*>(srow + col0);
#pragma unroll
              for (int v = 0; v < 8; ++v)
                dst[v] = make_float4(__uint_as_float(v32[4 * v]), __uint_as_float(v32[4 * v + 1]),
                                     __uint_as_float(v32[4 * v + 2]),
                                     __uint_as_float(v32[4 * v + 3]));
            } else {
#pragma unroll
              for (int i = 0; i < 32; ++i)
                if (col0 + i < p.n_valid) srow[col0 + i] = __uint_as_float(v32[i]);
            }
          }
        }
      } else if (MODE == kModeSwiGLU) {
#pragma unroll 1
        for (int c = 0; c < BN / 2; c += 32) {
          uint32_t g[32], u[32];
          tmem_ld32(tbase + c, g);
          tmem_ld32(tbase + BN / 2 + c, u);
          tmem_ld_wait();
          if (store) {
            uint32_t packed[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              const float g0 = __uint_as_float(g[2 * i]), g1 = __uint_as_float(g[2 * i + 1]);
              const float u0 = __uint_as_float(u[2 * i]), u1 = __uint_as_float(u[2 * i + 1]);
              const float a0 = g0 / (1.0f + __expf(-g0)) * u0;
              const float a1 = g1 / (1.0f + __expf(-g1)) * u1;
              __nv_bfloat162 h2 = __floats2bfloat162_rn(a0, a1);
              packed[i] = *reinterpret_cast<uint32_t*>(&h2);
            }
            uint4* dst = reinterpret_cast<uint4*>(orow + tl.n * (BN / 2) + c);
#pragma unroll
            for (int v = 0; v < 4; ++v)
              dst[v] = make_uint4(packed[4 * v], packed[4 * v + 1], packed[4 * v + 2],
                                  packed[4 * v + 3]);
          }
        }
      } else {
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          uint32_t v32[32];
          tmem_ld32(tbase + c, v32);
          tmem_ld_wait();
          if (store) {
            uint32_t packed[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              __nv_bfloat162 h2 = __floats2bfloat162_rn(__uint_as_float(v32[2 * i]),
                                                        __uint_as_float(v32[2 * i + 1]));
              packed[i] = *reinterpret_cast<uint32_t*>(&h2);
            }
            uint4* dst = reinterpret_cast<uint4*>(orow + tl.n * BN + c);
#pragma unroll
            for (int v = 0; v < 4; ++v)
              dst[v] = make_uint4(packed[4 * v], packed[4 * v + 1], packed[4 * v + 2],
                                  packed[4 * v + 3]);
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive1(smem_addr(&acc_empty[ab]));
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem_base, C::kTmemCols);
  }
  if (p.defer_wait) grid_dep_wait();
}

template <int BN, int MODE>
cudaError_t launch_impl(const TcGemmArgs& a, cudaStream_t stream) {
  using C = Cfg<BN>;
  auto kernel = grouped_gemm_kernel<BN, MODE>;
  cudaError_t e = cudaFuncSetAttribute(
      kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes);
  if (e != cudaSuccess) return e;
  KParams p;
  p.K = a.K;
  p.n_tiles = MODE == kModeSwiGLU ? a.n_total / (BN / 2) : a.n_total / BN;
  p.b_rows_per_group = a.b_rows_per_group;
  p.b_up_offset = a.b_up_offset;
  p.g = a.g;
  p.max_mtiles = a.g.offsets ? (a.g.cap_rows + BM - 1) / BM + a.g.E
                             : (a.g.dense_rows + BM - 1) / BM;
  p.out = static_cast<__nv_bfloat16*>(a.out);
  p.ldo = a.ldo;
  p.err = a.err;
  p.mt_prefix = a.g.mt_prefix;
  p.tile_rows = BM;
  p.k_splits = 1;
  p.out_f32 = nullptr;
  p.split_stride = 0;
  p.n_valid = 0;
  p.defer_wait = 0;
  p.b3d = MODE == kModeSwiGLU && a.b_gate_up_3d ? 1 : 0;
  p.norm_out = nullptr;
  p.tma_out = 0;
  p.gather_perm = nullptr;
  p.gather_kmax = 1;
  p.gather_tokens = 0;
  const int64_t max_tiles = static_cast<int64_t>(p.n_tiles) * p.max_mtiles;
  if (max_tiles == 0) return cudaSuccess;
  const int grid = static_cast<int>(max_tiles < a.num_sms ? max_tiles : a.num_sms);
  return launch_pdl(kernel, dim3(grid), dim3(kThreads), C::kSmemBytes, stream, *a.map_a,
                    *a.map_b, p);
}

// ===========================================================================
// 2-SM variant (cta_group::2) for groups of many rows.
//
// A cluster of two CTAs on one TPC computes a 256 x 256 tile: CTA rank r
// holds rows [row0 + 128 r, +128) of A and one half of the weight tile
// (SwiGLU: rank 0 the 128 gate rows, rank 1 the 128 matching up rows; down:
// rows n*256 + 128 r of W_down), so each SM streams 32 KB per 64-k block
// instead of 48 KB; the 192 KB ring holds 3 stages of two consecutive 64-k
// blocks.  With gathered rows (SwiGLU, TcGemmArgs::gather_perm) the A rows
// come straight from the token rows: every lane of the producer warp issues
// one four-row TMA gather per 64-k block, the tokens looked up through the
// pair permutation once per tile; the rows, tiles and MMA order are those of
// the copied rows, so the outputs are the same bits.  One thread of the
// leader CTA (rank 0) issues tcgen05.mma.cta_group::2 (M = 256, N = 256);
// each CTA's TMEM receives its 128 rows x 256 fp32 columns (two buffers of
// 256 columns, allocated collectively by one warp per CTA).
// Barriers: both producers arrive (with their byte counts) on the leader's
// "full" barrier and their TMA loads complete on it; MMA completion is
// multicast to both CTAs' "empty" and "accumulator full" barriers; both
// CTAs' epilogue warps arrive on the leader's "accumulator empty" barrier.
// Every barrier wait is bounded, as in the 1-SM kernel.
// ===========================================================================
// warps: 0 TMA producer, 1 MMA issuer (leader), 2-9 epilogue (two warps per
// TMEM lane quarter, each draining half of the accumulator's columns)
constexpr int kThreads2 = 320;
constexpr int kEpiWarps2 = 8;

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\t"
               "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// shared::cta address -> the same variable's shared::cluster address in CTA `rank`
__device__ __forceinline__ uint32_t map_to_rank(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}
// Byte-count announcement on the leader's barrier from the peer CTA: no
// release needed (the bytes themselves arrive by TMA complete_tx).
__device__ __forceinline__ void mbar_expect_tx_cluster(uint32_t cl_bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.relaxed.cluster.shared::cluster.b64 _, [%0], %1;" ::"r"(cl_bar),
               "r"(bytes)
               : "memory");
}
// Arrival that orders nothing but the arriving thread's own progress: used to
// hand a TMEM accumulator back once its last tcgen05.ld has completed
// (tcgen05.wait::ld); the epilogue's global stores need not be visible to
// the MMA issuer, so no release fence makes them drain first.
__device__ __forceinline__ void mbar_arrive_cluster_relaxed(uint32_t cl_bar) {
  asm volatile("mbarrier.arrive.relaxed.cluster.shared::cluster.b64 _, [%0];" ::"r"(cl_bar)
               : "memory");
}
// TMA tile load whose completion is counted on a barrier in either CTA of the pair.
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap* map, int c0,
                                                 int c1, uint32_t cl_bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.cta_group::2"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(cl_bar)
      : "memory");
}
// Four rows r0..r3 of a map whose box is {64, 1}, copied to four consecutive
// 128-byte rows at dst (the same 128-byte swizzle as a tiled box: it follows
// the shared-memory address, and dst is 512-byte aligned, half of an 8-row
// swizzle atom), completion counted on a barrier in either CTA of the pair.
__device__ __forceinline__ void tma_gather4_pair(uint32_t dst, const CUtensorMap* map, int c0,
                                                 const int (&r)[4], uint32_t cl_bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile::gather4.mbarrier::complete_tx::bytes"
      ".cta_group::2 [%0], [%1, {%2, %3, %4, %5, %6}], [%7];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]),
      "r"(cl_bar)
      : "memory");
}
__device__ __forceinline__ void mma_bf16_pair(uint32_t tmem_d, uint64_t da, uint64_t db,
                                              uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(tmem_d),
      "l"(da), "l"(db), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive on the barrier at this shared-memory offset in both CTAs of the pair
// once all prior MMAs of this thread have completed.
__device__ __forceinline__ void mma_commit_pair(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(bar),
      "h"(static_cast<uint16_t>(0x3))
      : "memory");
}
__device__ __forceinline__ void tmem_alloc_pair(uint32_t slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(slot),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}

struct Cfg2 {
  static constexpr int BN = 256;                 // output tile width of the pair
  static constexpr int KS = 2;                   // 64-k blocks per stage
  static constexpr int kSubBytes = BM * BK * 2;  // 16 KB: one 128-row x 64-k box
  static constexpr int kABytes = KS * kSubBytes; // this CTA's 128 rows
  static constexpr int kBBytes = KS * kSubBytes; // this CTA's half of the weight tile
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kStages = kRingBytes / kStageBytes;  // 3
  static constexpr int kTmemCols = 2 * BN;       // two accumulators
  static constexpr int kStagingBytes = 32 * 128; // per epilogue warp: 32 rows x 128 B
  static constexpr int kIndexInts = 384;         // both prefix arrays to E = 191, the first to 383
  static constexpr int kSmemBytes =
      kStages * kStageBytes + 256 + kEpiWarps2 * kStagingBytes + kIndexInts * 4 + 1024;
  static_assert(kSmemBytes <= 227 * 1024, "shared memory of one CTA");
};

// TMA tile store of a shared-memory box (bulk-group completion) and its waits.
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, uint32_t src, int c0,
                                             int c1) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];"
               ::"l"(reinterpret_cast<uint64_t>(map)), "r"(src), "r"(c0), "r"(c1)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() {
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
// the stores issued so far have read their shared-memory source
__device__ __forceinline__ void bulk_wait_read() {
  asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
// ... and completed
__device__ __forceinline__ void bulk_wait_all() {
  asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}

// The epilogue's bf16 rows reach global memory through a per-warp staging
// tile: each thread writes its row's 128 bytes (16-byte chunk j at position
// j ^ (row & 7), so the 32 rows' writes spread over the banks), then each
// store instruction of the warp writes four whole 128-byte row segments
// (lane l: row 4 i + l / 8, chunk l % 8).  Per-lane stores of 16 bytes to 32
// different rows cost one L2 request per 16 bytes, as many requests as the
// TMA loads of the main loop; this costs one per 128 bytes.
__device__ __forceinline__ void stage_chunk(uint8_t* stg, int lane, int j, const uint4& v) {
  *reinterpret_cast<uint4*>(stg + lane * 128 + ((j ^ (lane & 7)) << 4)) = v;
}
// rows [0, nrows) of the staging tile to out rows row_base + r, columns
// col0 .. col0 + 63 (bf16), row stride ldo
__device__ __forceinline__ void flush_staging(const uint8_t* stg, int lane,
                                              __nv_bfloat16* out, int64_t row_base, int ldo,
                                              int col0, int nrows) {
  __syncwarp();
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int r = 4 * i + (lane >> 3), c = lane & 7;
    const uint4 v = *reinterpret_cast<const uint4*>(stg + r * 128 + ((c ^ (r & 7)) << 4));
    if (r < nrows)
      *reinterpret_cast<uint4*>(out + (row_base + r) * ldo + col0 + 8 * c) = v;
  }
  __syncwarp();
}

template <int MODE>
__global__ void __launch_bounds__(kThreads2, 1)
    grouped_gemm_pair_kernel(const __grid_constant__ CUtensorMap map_a,
                             const __grid_constant__ CUtensorMap map_b,
                             const __grid_constant__ CUtensorMap map_out, const KParams p) {
  using C = Cfg2;
  constexpr int kStages = C::kStages;
  constexpr int BN = C::BN;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* sa = smem;
  uint8_t* sb = smem + kStages * C::kABytes;
  // after the ring: the epilogue warps' staging tiles (1024-byte aligned,
  // the 128-byte swizzle of the output map), the barriers, the tile index
  uint8_t* staging = smem + kStages * C::kStageBytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(staging + kEpiWarps2 * C::kStagingBytes);
  uint64_t* full = bars;                        // leader's is the one used
  uint64_t* empty = bars + kStages;             // per CTA
  uint64_t* acc_full = bars + 2 * kStages;      // per CTA
  uint64_t* acc_empty = bars + 2 * kStages + 2; // leader's is the one used
  uint64_t* drain = bars + 2 * kStages + 4;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * kStages + 5);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();
  const bool leader = rank == 0;
  const int pair = blockIdx.x >> 1;
  const int npairs = gridDim.x >> 1;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 2);  // one expect_tx arrival per CTA of the pair
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], 2 * kEpiWarps2);  // every epilogue warp of both CTAs
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_map(&map_a);
    prefetch_map(&map_b);
    if (p.tma_out) prefetch_map(&map_out);
  }
  cluster_sync_all();  // barriers of both CTAs initialised; the peer is running
  if (warp == 1) tmem_alloc_pair(smem_addr(tmem_slot), C::kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  grid_dep_wait();
  grid_dep_launch();
  const TileIndex ix =
      load_tile_index(p, reinterpret_cast<int32_t*>(reinterpret_cast<uint8_t*>(bars) + 256),
                      C::kIndexInts);
  // tiles are 256 rows (both CTAs) x 256 columns; mt_prefix counts 256-row tiles
  const int ntiles = total_tiles(p, ix);
  const int nk = p.K / (BK * C::KS);  // stages per tile

  // SwiGLU with gathered A rows: the whole producer warp issues the A
  // copies, one four-row gather per lane and 64-k block (lane l: rows 4 l ..
  // 4 l + 3 of this CTA's 128); otherwise lane 0 issues everything
  const bool gather = MODE == kModeSwiGLU && p.gather_perm != nullptr;
  if (warp == 0 && (gather || lane == 0)) {
    // ---------------- TMA producer (each CTA: its A rows, its B half) -------
    int stage = 0;
    uint32_t phase = 0;
    uint32_t issued_mask = 0, issued_phase = 0;
    bool ok = true;
    for (int t = pair; t < ntiles && ok; t += npairs) {
      Tile tl;
      if (!decode_tile(p, ix, t, tl)) {  // the same outcome in every lane
        if (lane == 0) {
          set_err(p.err, kErrIndex);
          *abort_flag = 1;
        }
        break;
      }
      // token of each of this lane's four rows; rows past the tile's end
      // repeat its last row (computed, never stored)
      int tok[4] = {0, 0, 0, 0};
      if (gather) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int r = min(static_cast<int>(rank) * BM + 4 * lane + i, tl.rows - 1);
          const int o = p.gather_perm[tl.row0 + r];
          const int tk = o >= 0 ? o / p.gather_kmax : -1;
          if (tk < 0 || tk >= p.gather_tokens)
            set_err(p.err, kErrIndex);
          else
            tok[i] = tk;
        }
      }
      for (int kb = 0; kb < nk; ++kb) {
        // every issuing lane observes the stage's release itself
        const bool w = mbar_wait(&empty[stage], phase ^ 1u, abort_flag, kWaitNs);
        if (!(gather ? __all_sync(0xffffffffu, w) : w)) {
          ok = false;
          break;
        }
        const uint32_t fb = map_to_rank(smem_addr(&full[stage]), 0);
        int brow;
        if (MODE == kModeSwiGLU)
          brow = tl.e * p.b_rows_per_group + (rank ? p.b_up_offset : 0) + tl.n * (BN / 2);
        else
          brow = tl.e * p.b_rows_per_group + tl.n * BN + static_cast<int>(rank) * (BN / 2);
        if (lane == 0) {
          if (leader)
            mbar_expect_tx(smem_addr(&full[stage]), C::kStageBytes);
          else
            mbar_expect_tx_cluster(fb, C::kStageBytes);
          // consecutive k blocks of the same rows back to back
#pragma unroll
          for (int u = 0; u < C::KS; ++u) {
            const int k0 = (kb * C::KS + u) * BK;
            if (!gather)
              tma_load_2d_pair(smem_addr(sa + stage * C::kABytes + u * C::kSubBytes), &map_a,
                               k0, tl.row0 + static_cast<int>(rank) * BM, fb);
            tma_load_2d_pair(smem_addr(sb + stage * C::kBBytes + u * C::kSubBytes), &map_b, k0,
                             brow, fb);
          }
        }
        if (gather) {
          __syncwarp();
#pragma unroll
          for (int u = 0; u < C::KS; ++u)
            tma_gather4_pair(
                smem_addr(sa + stage * C::kABytes + u * C::kSubBytes + lane * 4 * 128), &map_a,
                (kb * C::KS + u) * BK, tok, fb);
        }
        issued_mask |= 1u << stage;
        issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
        if (++stage == kStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
    if (lane == 0) {
      if (!ok) {
        set_err(p.err, kErrTimeout);
        *abort_flag = 1;
      }
      if (*abort_flag && leader) {
        for (int s = 0; s < kStages; ++s)
          if (issued_mask & (1u << s))
            mbar_wait(&full[s], (issued_phase >> s) & 1u, nullptr, kDrainNs);
      }
    }
  } else if (warp == 1 && lane == 0 && leader) {
    // ---------------- MMA issuer (leader CTA only) ----------------
    constexpr uint32_t idesc = (1u << 4) | (1u << 7) | (1u << 10) |
                               (static_cast<uint32_t>(BN >> 3) << 17) |
                               (static_cast<uint32_t>((2 * BM) >> 4) << 24);
    int stage = 0;
    uint32_t phase = 0;
    int lt = 0;
    bool ok = true, issued_any = false;
    for (int t = pair; t < ntiles && ok; t += npairs, ++lt) {
      const int ab = lt & 1;
      const uint32_t acc_phase = (lt >> 1) & 1;
      if (!mbar_wait(&acc_empty[ab], acc_phase ^ 1u, abort_flag, kWaitNs)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(ab * BN);
      for (int kb = 0; kb < nk; ++kb) {
        if (!mbar_wait(&full[stage], phase, abort_flag, kWaitNs)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a0 = smem_addr(sa + stage * C::kABytes);
        const uint32_t b0 = smem_addr(sb + stage * C::kBBytes);
#pragma unroll
        for (int u = 0; u < C::KS; ++u)
#pragma unroll
          for (int k = 0; k < BK / UMMA_K; ++k)
            mma_bf16_pair(d_tmem, desc_sw128(a0 + u * C::kSubBytes + k * UMMA_K * 2),
                          desc_sw128(b0 + u * C::kSubBytes + k * UMMA_K * 2), idesc,
                          (kb > 0 || u > 0 || k > 0) ? 1u : 0u);
        issued_any = true;
        mma_commit_pair(smem_addr(&empty[stage]));
        if (++stage == kStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
      if (!ok) break;
      mma_commit_pair(smem_addr(&acc_full[ab]));
    }
    if (!ok) {
      set_err(p.err, kErrTimeout);
      *abort_flag = 1;
    }
    if (*abort_flag && issued_any) {
      mma_commit_pair(smem_addr(drain));
      mbar_wait(drain, 0, nullptr, kDrainNs);
    }
  } else if (warp >= 2) {
    // ---------------- epilogue (each CTA: its 128 rows) ----------------
    // warp w drains TMEM lanes 32 (w % 4) .. +31 (its quarter of the rows)
    // and one half of the columns: warps 2-5 the first, 6-9 the second.
    // The TMEM loads of a half are issued two chunks at a time before one
    // wait; once the last chunk is in registers the accumulator is handed
    // back (relaxed arrive), and the conversion and stores of that chunk
    // overlap the next tile's MMAs.
    const int quarter = warp & 3;
    const int half = (warp - 2) >> 2;
    const int wrow0 = static_cast<int>(rank) * BM + quarter * 32;  // warp's first row in the 256
    uint8_t* stg = staging + (warp - 2) * C::kStagingBytes;
    // Whole 32-row chunks leave by one TMA store of the staging tile (the
    // store engine writes the lines; per-lane stores of the same lines cost
    // the down GEMM of the 32 x 1024 layer about 57 us of its 455); a chunk
    // that ends inside the tile's group keeps the per-lane stores, which
    // stop at its last row.  The tile is rewritten only after the previous
    // store has read it.
    const bool tma_out = p.tma_out != 0;
    auto staging_free = [&]() {
      if (tma_out) {
        if (lane == 0) bulk_wait_read();
        __syncwarp();
      }
    };
    auto emit = [&](int64_t rbase, int col0, int nrows) {
      if (tma_out && nrows == 32) {
        fence_proxy_async_smem();  // this lane's staging writes, before the store reads them
        __syncwarp();
        if (lane == 0) {
          tma_store_2d(&map_out, smem_addr(stg), col0, static_cast<int>(rbase));
          bulk_commit();
        }
      } else {
        flush_staging(stg, lane, p.out, rbase, p.ldo, col0, nrows);
      }
    };
    const uint32_t acc_empty_leader0 = map_to_rank(smem_addr(&acc_empty[0]), 0);
    const uint32_t acc_empty_leader1 = map_to_rank(smem_addr(&acc_empty[1]), 0);
    int lt = 0;
    for (int t = pair; t < ntiles; t += npairs, ++lt) {
      Tile tl;
      const bool tile_ok = decode_tile(p, ix, t, tl);
      const int ab = lt & 1;
      const uint32_t acc_phase = (lt >> 1) & 1;
      int ok = 1;
      if (lane == 0) ok = mbar_wait(&acc_full[ab], acc_phase, abort_flag, kWaitNs) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) {
        if (lane == 0) {
          if (!*abort_flag) set_err(p.err, kErrTimeout);
          *abort_flag = 1;
        }
        break;
      }
      tc_fence_after();
      const uint32_t tbase = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) +
                             static_cast<uint32_t>(ab * BN);
      // rows of this warp that belong to the tile (0 when the tile is bad)
      const int nrows = tile_ok ? max(0, min(32, tl.rows - wrow0)) : 0;
      const int64_t row_base = static_cast<int64_t>(tl.row0) + wrow0;
      const uint32_t release_bar = ab ? acc_empty_leader1 : acc_empty_leader0;
      auto hand_back = [&]() {
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster_relaxed(release_bar);
      };
      if (MODE == kModeSwiGLU) {
        // output columns [64 half, +64): gate at c, up at BN/2 + c; both
        // 32-column rounds fill one 128-byte staging row
        staging_free();
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          const int c = half * 64 + 32 * r;
          uint32_t g[32], u[32];
          tmem_ld32(tbase + c, g);
          tmem_ld32(tbase + BN / 2 + c, u);
          tmem_ld_wait();
          if (r == 1) hand_back();
          uint32_t packed[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const float g0 = __uint_as_float(g[2 * i]), g1 = __uint_as_float(g[2 * i + 1]);
            const float u0 = __uint_as_float(u[2 * i]), u1 = __uint_as_float(u[2 * i + 1]);
            const float a0 = g0 / (1.0f + __expf(-g0)) * u0;
            const float a1 = g1 / (1.0f + __expf(-g1)) * u1;
            __nv_bfloat162 h2 = __floats2bfloat162_rn(a0, a1);
            packed[i] = *reinterpret_cast<uint32_t*>(&h2);
          }
#pragma unroll
          for (int v = 0; v < 4; ++v)
            stage_chunk(stg, lane, 4 * r + v,
                        make_uint4(packed[4 * v], packed[4 * v + 1], packed[4 * v + 2],
                                   packed[4 * v + 3]));
        }
        emit(row_base, tl.n * (BN / 2) + half * 64, nrows);
      } else {
        // columns [128 half, +128) in two rounds of 64 (one staging row each)
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          const int c = half * 128 + 64 * r;
          uint32_t v0[32], v1[32];
          tmem_ld32(tbase + c, v0);
          tmem_ld32(tbase + c + 32, v1);
          tmem_ld_wait();
          if (r == 1) hand_back();
          uint32_t packed[32];
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            __nv_bfloat162 h0 = __floats2bfloat162_rn(__uint_as_float(v0[2 * i]),
                                                      __uint_as_float(v0[2 * i + 1]));
            __nv_bfloat162 h1 = __floats2bfloat162_rn(__uint_as_float(v1[2 * i]),
                                                      __uint_as_float(v1[2 * i + 1]));
            packed[i] = *reinterpret_cast<uint32_t*>(&h0);
            packed[16 + i] = *reinterpret_cast<uint32_t*>(&h1);
          }
          staging_free();
#pragma unroll
          for (int v = 0; v < 8; ++v)
            stage_chunk(stg, lane, v,
                        make_uint4(packed[4 * v], packed[4 * v + 1], packed[4 * v + 2],
                                   packed[4 * v + 3]));
          emit(row_base, tl.n * BN + c, nrows);
        }
      }
    }
    if (tma_out && lane == 0) bulk_wait_all();  // every store written before exit
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // the pair's MMAs and TMEM reads are done in both CTAs
  tc_fence_after();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc_pair(tmem_base, C::kTmemCols);
  }
}

template <int MODE>
cudaError_t launch_pair_impl(const TcGemmArgs& a, cudaStream_t stream) {
  using C = Cfg2;
  auto kernel = grouped_gemm_pair_kernel<MODE>;
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       C::kSmemBytes);
  if (e != cudaSuccess) return e;
  if (a.K % (BK * C::KS) != 0) return cudaErrorInvalidValue;  // whole stages
  KParams p;
  p.K = a.K;
  p.n_tiles = MODE == kModeSwiGLU ? a.n_total / (C::BN / 2) : a.n_total / C::BN;
  p.b_rows_per_group = a.b_rows_per_group;
  p.b_up_offset = a.b_up_offset;
  p.g = a.g;
  p.mt_prefix = a.g.mt2_prefix;
  p.tile_rows = 2 * BM;
  p.max_mtiles = a.g.offsets ? (a.g.cap_rows + p.tile_rows - 1) / p.tile_rows + a.g.E
                             : (a.g.dense_rows + p.tile_rows - 1) / p.tile_rows;
  p.out = static_cast<__nv_bfloat16*>(a.out);
  p.ldo = a.ldo;
  p.err = a.err;
  p.k_splits = 1;
  p.out_f32 = nullptr;
  p.split_stride = 0;
  p.n_valid = 0;
  p.defer_wait = 0;
  p.b3d = 0;
  p.norm_out = nullptr;
  p.tma_out = a.map_out != nullptr ? 1 : 0;
  p.gather_perm = MODE == kModeSwiGLU ? a.gather_perm : nullptr;
  p.gather_kmax = a.gather_kmax;
  p.gather_tokens = a.gather_tokens;
  if (p.gather_perm != nullptr && (p.gather_kmax < 1 || p.gather_tokens < 1))
    return cudaErrorInvalidValue;
  const int64_t max_tiles = static_cast<int64_t>(p.n_tiles) * p.max_mtiles;
  if (max_tiles == 0) return cudaSuccess;
  int pairs = a.num_sms / 2;
  if (pairs > max_tiles) pairs = static_cast<int>(max_tiles);
  if (pairs < 1) pairs = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * pairs);
  cfg.blockDim = dim3(kThreads2);
  cfg.dynamicSmemBytes = C::kSmemBytes;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  // without an output map the per-lane stores run and map_a stands in
  return cudaLaunchKernelEx(&cfg, kernel, *a.map_a, *a.map_b,
                            a.map_out != nullptr ? *a.map_out : *a.map_a, p);
}

}  // namespace

cudaError_t launch_swiglu_tc(const TcGemmArgs& a, int bn, cudaStream_t stream) {
  if (bn == 128) return launch_impl<128, kModeSwiGLU>(a, stream);
  return launch_impl<256, kModeSwiGLU>(a, stream);
}
cudaError_t launch_down_tc(const TcGemmArgs& a, int bn, cudaStream_t stream) {
  if (bn == 128) return launch_impl<128, kModeDown>(a, stream);
  return launch_impl<256, kModeDown>(a, stream);
}
template <int BN>
cudaError_t launch_scores_impl(const TcGemmArgs& a, int k_splits, float* out,
                               int64_t split_stride, int n_valid, bool defer_wait,
                               float* row_norms, cudaStream_t stream) {
  using C = Cfg<BN>;
  auto kernel = grouped_gemm_kernel<BN, kModeScores>;
  if (a.g.offsets != nullptr || k_splits < 1 || (a.K / BK) % k_splits != 0 ||
      a.K % BK != 0 || n_valid < 1 || (row_norms != nullptr && k_splits != 1))
    return cudaErrorInvalidValue;
  cudaError_t e = cudaFuncSetAttribute(
      kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes);
  if (e != cudaSuccess) return e;
  KParams p{};
  p.K = a.K;
  p.n_tiles = (n_valid + BN - 1) / BN;
  p.b_rows_per_group = 0;
  p.b_up_offset = 0;
  p.g = a.g;
  p.max_mtiles = (a.g.dense_rows + BM - 1) / BM;
  p.out = nullptr;
  p.ldo = a.ldo;
  p.err = a.err;
  p.mt_prefix = nullptr;
  p.tile_rows = BM;
  p.k_splits = k_splits;
  p.out_f32 = out;
  p.split_stride = split_stride;
  p.n_valid = n_valid;
  p.defer_wait = defer_wait ? 1 : 0;
  p.b3d = 0;
  p.norm_out = row_norms;
  const int64_t max_tiles = static_cast<int64_t>(p.n_tiles) * p.max_mtiles * k_splits;
  if (max_tiles == 0) return cudaSuccess;
  const int grid = static_cast<int>(max_tiles < a.num_sms ? max_tiles : a.num_sms);
  return launch_pdl(kernel, dim3(grid), dim3(kThreadsScores), C::kSmemBytes, stream,
                    *a.map_a, *a.map_b, p);
}

// SwiGLU loads gate and up halves as two boxes of bn/2 rows; down loads one
// box of bn rows.
int tc_b_box_rows(bool swiglu, int bn) { return swiglu ? bn / 2 : bn; }

cudaError_t launch_scores_tc(const TcGemmArgs& a, int bn, int k_splits, float* out,
                             int64_t split_stride, int n_valid, bool defer_wait,
                             cudaStream_t stream, float* row_norms) {
  if (bn == 64)
    return launch_scores_impl<64>(a, k_splits, out, split_stride, n_valid, defer_wait,
                                  row_norms, stream);
  if (bn == 128)
    return launch_scores_impl<128>(a, k_splits, out, split_stride, n_valid, defer_wait,
                                   row_norms, stream);
  return cudaErrorInvalidValue;
}

cudaError_t launch_swiglu_tc_pair(const TcGemmArgs& a, cudaStream_t stream) {
  return launch_pair_impl<kModeSwiGLU>(a, stream);
}
cudaError_t launch_down_tc_pair(const TcGemmArgs& a, cudaStream_t stream) {
  return launch_pair_impl<kModeDown>(a, stream);
}
// Output columns of one tile.
int tc_n_granule(bool swiglu, int bn) { return swiglu ? bn / 2 : bn; }

// Tile width: 256 when there are enough tiles to fill every SM several
// times over (large M per expert: fewer re-reads of the A rows per output),
// else 128 so that the persistent CTAs get more, smaller tiles and the last
// partial wave is short (small M: the GEMM is a weight stream).
int tc_pick_bn(bool swiglu, int n_total, int64_t mtiles_est, int num_sms) {
  const int g256 = tc_n_granule(swiglu, 256);
  const int g128 = tc_n_granule(swiglu, 128);
  if (n_total % g256 != 0) return (n_total % g128 == 0) ? 128 : 0;
  const int64_t tiles256 = static_cast<int64_t>(n_total / g256) * mtiles_est;
  return tiles256 >= 8LL * num_sms ? 256 : 128;
}

}  // namespace rx
