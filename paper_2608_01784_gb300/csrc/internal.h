// internal.h — launchers shared between the kernel files and the C-ABI host
// code (reflex_abi.cu).  Not part of the public ABI.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace rx {

struct AllocArgs {
  int k_min, k_base, k_max, delta_role, delta_cur;
  float q, theta, w_cf, v_ref, tau;
  int signal;             // rank key of the Eq. 9 groups (REFLEX_SIGNAL_*)
  int role_shuffle;       // permute each sequence's final counts
  uint64_t shuffle_seed;  // splitmix64 seed of the permutation keys
  int count_rule;         // REFLEX_RULE_*: 0 = this allocation, else a score rule
  float rule_threshold;   // p of Top-p / the expert-threshold router weight
};

// ---- allocation (budget.cu) -----------------------------------------------
// alongside: launched right after a kernel that writes none of the inputs
// (the router scores of the same forward), with err / k_sum already cleared
// when B > 1; the counts then run next to that kernel, and the budget grid
// still completes only after it.
cudaError_t launch_budget(const float* conf1, const float* conf2,
                          const uint8_t* hist_len, const uint8_t* masked,
                          const int32_t* block_id, const int32_t* seq_off,
                          const int32_t* active_block, int T, int B,
                          const AllocArgs& a, int32_t* k_out,
                          unsigned long long* k_sum, uint32_t* err,
                          cudaStream_t stream, bool alongside = false);
cudaError_t launch_wait_selftest(uint32_t* err, uint64_t limit_ns,
                                 cudaStream_t stream);

// ---- refinement-state update (state.cu) ------------------------------------
cudaError_t launch_update_state(const float* conf_new, float* conf1, float* conf2,
                                uint8_t* hist_len, uint8_t* masked, const int32_t* block_id,
                                const int32_t* seq_off, int32_t* active,
                                const int32_t* num_blocks, int T, int B, float theta,
                                int32_t* committed, uint32_t* err, cudaStream_t stream);

// ---- routing (router.cu) --------------------------------------------------
// z[T, E] = router scores (sequential fp32 fma chain over the hidden index).
// The first CTA also clears zero_words[0, n_zero) (nullable): the call's
// header or error word, so no memset precedes the first kernel.  err
// (nullable) receives kErrTimeout if a bounded wait of a kernel expires.
// pf (optional): bytes the score kernel hands to the L2 as bulk prefetches
// while it computes (the next kernels' weights; HBM is otherwise idle then).
struct L2Prefetch {
  const void* base = nullptr;
  uint64_t bytes = 0;  // a multiple of 16
};
cudaError_t launch_router_logits(int dtype, const void* hidden,
                                 const void* w_router, int T, int d, int E,
                                 float* z, uint32_t* zero_words, int n_zero,
                                 uint32_t* err, int num_sms, cudaStream_t stream,
                                 const L2Prefetch& pf = L2Prefetch{});
// Screened routing (bf16, renormalised weights): nw[e] = ||w_e||_2 rounded up
// (first kernel of the forward; clears zero_words like the score kernels);
// then, from the tensor-core score slices z[s][t][e] (s < k_splits), the
// exact TopK, alpha and ids, with the canonical chain recomputed for every
// expert that could be selected (written back into z's first slice).
cudaError_t launch_router_wnorm(const __nv_bfloat16* w, int E, int d, float* nw,
                                uint32_t* zero_words, int n_zero, cudaStream_t stream);
cudaError_t launch_router_screen_select(const __nv_bfloat16* h, const __nv_bfloat16* w,
                                        float* z, int k_splits, int64_t split_stride,
                                        const float* nw, const int32_t* k, int T, int E,
                                        int d, int k_max, int32_t* ids, float* alpha,
                                        uint32_t* err, cudaStream_t stream);
// Tile width and K slices of the screen GEMM for T x E scores over d: slices
// double while the tile count stays within 152 (this GPU's SM count).
inline int screen_bn(int E) { return E <= 64 ? 64 : 128; }
inline int screen_splits(int T, int E, int d) {
  const int64_t mt = (T + 127) / 128, nt = (E + screen_bn(E) - 1) / screen_bn(E);
  const int nkb = d / 64;
  int s = 1;
  while (s < 16 && mt * nt * s * 2 <= 152 && nkb % (2 * s) == 0) s *= 2;
  return s;
}
// Rows of the workspace's score region for the screen GEMM's slices: s T,
// and never fewer than for a smaller batch (s falls as T adds tiles, and a
// workspace sized for a batch must serve every smaller one).  A batch of m
// full 128-row tiles has the most rows among those of m tiles; beyond 152
// tiles s = 1.
inline int64_t screen_z_rows(int T, int E, int d) {
  int64_t rows = static_cast<int64_t>(screen_splits(T, E, d)) * T;
  const int64_t mt = (T + 127) / 128;
  for (int64_t m = 1; m < mt && m <= 152; ++m) {
    const int64_t r = screen_splits(static_cast<int>(m * 128), E, d) * m * 128;
    if (r > rows) rows = r;
  }
  return rows;
}
// Batched screen for E <= 256 (bf16, renormalised weights): z holds the
// tensor-core estimates [T, E] (one K slice), hss the tokens' sums of
// squares, nw the experts' norms (wnorm_kernel); map_h / map_w are 2D maps of
// the hidden states [T, d] and the router weights [E, d] with boxes of 64
// columns and screen_batch_token_rows(E) / screen_batch_expert_rows(E) rows (128-byte
// swizzle).  Writes ids / alpha and the candidates' exact scores into z.
// the box heights of map_h (tokens per CTA) and map_w for E experts
int screen_batch_token_rows(int E);
int screen_batch_expert_rows(int E);
cudaError_t launch_router_screen_batch(const CUtensorMap* map_h, const CUtensorMap* map_w,
                                       float* z, const float* hss, const float* nw,
                                       const int32_t* k, int T, int E, int d, int k_max,
                                       int32_t* ids, float* alpha, uint32_t* err,
                                       cudaStream_t stream);
// The counts from the router scores (count rules 1 = Top-p, 2 = expert
// threshold, threshold thr, clip [k_lo, min(k_hi, E)]) into k_out (and added
// to k_sum, nullable, which the caller cleared), then ids / alpha [T, k_max]
// as launch_router_select gives them for those counts; ids == nullptr:
// counts only.
cudaError_t launch_router_select_rule(const float* z, int T, int E, int k_hi, int k_lo,
                                      int rule, float thr, int k_max, bool renorm,
                                      int32_t* k_out, unsigned long long* k_sum,
                                      int32_t* ids, float* alpha, cudaStream_t stream);
// ids/alpha [T, k_max] from z and the counts k.
cudaError_t launch_router_select(const float* z, const int32_t* k, int T,
                                 int E, int k_max, bool renorm, int32_t* ids,
                                 float* alpha, uint32_t* err,
                                 cudaStream_t stream);

// ---- dispatch (dispatch.cu) -----------------------------------------------
struct DispatchBufs {
  int32_t* blk_count;  // [nblk, E]
  int32_t* blk_off;    // [nblk, E]
  int32_t* counts;     // [E]
  int32_t* offsets;    // [E+1]
  int32_t* mt_prefix;  // [E+1] 128-row tiles
  int32_t* mt2_prefix; // [E+1] 256-row tiles
  int32_t* perm;       // [T*k_max]
  int32_t* row_of;     // [T*k_max]
  int32_t* totals;     // header: total_pairs, total_mtiles, total_mtiles2
  uint32_t* err;
  uint32_t* blk_mask;  // [nblk, E, BLK / 32] token bits of each block and expert
};
constexpr int kDispatchBlock = 256;       // tokens per dispatch block, large batches
constexpr int kDispatchBlockSmall = 32;   // tokens per dispatch block up to 4096 tokens
constexpr int kDispatchSmallT = 4096;
inline int dispatch_block(int T) { return T <= kDispatchSmallT ? kDispatchBlockSmall : kDispatchBlock; }
// per-block count buffers sized for either block size (monotonic in T, so a
// workspace sized for a batch also fits every smaller one)
inline int64_t dispatch_blocks_alloc(int T) {
  const int ts = T < kDispatchSmallT ? T : kDispatchSmallT;
  return (ts + kDispatchBlockSmall - 1) / kDispatchBlockSmall +
         (T + kDispatchBlock - 1) / kDispatchBlock;
}
// The pair layout (counts, offsets, tile prefixes, perm, row_of) and the
// gathered rows X_perm[row_of[t, j]] = X[t] for j < k_t (x_perm nullptr:
// the layout only, for a consumer that gathers the rows itself).
// mask words for either block size (monotonic in T, like the block counts)
inline int64_t dispatch_mask_words_alloc(int T) {
  const int ts = T < kDispatchSmallT ? T : kDispatchSmallT;
  return (ts + kDispatchBlockSmall - 1) / kDispatchBlockSmall +
         static_cast<int64_t>(T + kDispatchBlock - 1) / kDispatchBlock * (kDispatchBlock / 32);
}
cudaError_t launch_dispatch_gather(int dtype, const void* hidden, const int32_t* ids,
                                   const int32_t* k, int T, int E, int k_max, int cap_rows,
                                   int d, const DispatchBufs& b, void* x_perm, int num_sms,
                                   cudaStream_t stream);

// ---- experts: SIMT grouped GEMMs (experts_simt.cu) ------------------------
// Grouped mode: rows [offsets[e], offsets[e+1]) use expert e; dense mode
// (offsets == nullptr): rows [0, dense_rows) use the single weight set.
struct GroupRows {
  const int32_t* offsets;    // [E+1] or nullptr
  const int32_t* mt_prefix;  // [E+1] prefix of 128-row tile counts
  const int32_t* mt2_prefix; // [E+1] prefix of 256-row tile counts
  const int32_t* totals;     // device total rows (grouped mode)
  int E;
  int dense_rows;
  int cap_rows;
};
cudaError_t launch_swiglu_simt(int dtype, const void* x, const void* w_gate_up,
                               int d, int inter, const GroupRows& g, void* act,
                               uint32_t* err, cudaStream_t stream);
cudaError_t launch_down_simt(int dtype, const void* act, const void* w_down,
                             int d, int inter, const GroupRows& g, void* y,
                             uint32_t* err, cudaStream_t stream);

// ---- experts: tcgen05 grouped GEMMs (experts_tc.cu) -----------------------
struct TcGemmArgs {
  const CUtensorMap* map_a;  // A [rows, K] bf16, box {64, 128}, 128B swizzle
  const CUtensorMap* map_b;  // B [groups * rows_per_group, K] bf16
  int K;                     // reduction length
  int n_total;               // output columns per group (SwiGLU: inter)
  int b_rows_per_group;      // SwiGLU: 2*inter, down: d
  int b_up_offset;           // SwiGLU: inter (row offset of up weights)
  GroupRows g;               // row groups
  void* out;                 // [rows, ldo] bf16
  int ldo;
  uint32_t* err;
  int num_sms;
  // SwiGLU, 1-SM kernel: map_b is the 3D map of tc_gate_up_3d (box {64,
  // bn / 2, 2}: a tile's gate and up rows in one copy) instead of a 2D map
  bool b_gate_up_3d = false;
  // SwiGLU, CTA-pair kernel: when set, map_a is a {64, 1}-box map of the
  // token rows X [gather_tokens, K], and A row r is token gather_perm[r] /
  // gather_kmax (row r's pair index over k_max), fetched by four-row TMA
  // gathers; nullptr: map_a holds the rows in pair order
  const int32_t* gather_perm = nullptr;
  int gather_kmax = 0;
  int gather_tokens = 0;
  // CTA-pair kernels: 2D map of out [rows, ldo] with a {64, 32} box, 128-byte
  // swizzle; whole 32-row output chunks are written by TMA stores through it
  // (nullptr: per-lane stores)
  const CUtensorMap* map_out = nullptr;
};
// SwiGLU: out = silu(A Wg^T) * (A Wu^T).  Down: out = A Wd^T.  bn = tile
// width (128 or 256, from tc_pick_bn); the B tensor map's box must have
// tc_b_box_rows(swiglu, bn) rows.
cudaError_t launch_swiglu_tc(const TcGemmArgs& a, int bn, cudaStream_t stream);
cudaError_t launch_down_tc(const TcGemmArgs& a, int bn, cudaStream_t stream);
int tc_b_box_rows(bool swiglu, int bn);
// Router-score screen: out[ks][t][e] = sum over the ks-th of k_splits equal
// slices of k of A[t, k] B[e, k] (fp32 accumulators, dense rows t < T =
// a.g.dense_rows, columns e < n_valid, row stride a.ldo), bn in {64, 128}
// (B tensor map box of bn rows); a.K / 64 must be a multiple of k_splits.
// defer_wait: launched right behind a kernel that writes none of its inputs
// or outputs (it then overlaps that kernel and waits for it before exiting).
// row_norms (nullable, k_splits == 1 only): the sum of squares of every A
// row (fp32, one per row), computed from the staged A tiles.
cudaError_t launch_scores_tc(const TcGemmArgs& a, int bn, int k_splits, float* out,
                             int64_t split_stride, int n_valid, bool defer_wait,
                             cudaStream_t stream, float* row_norms = nullptr);
// CTA-pair (2-SM, cta_group::2) variants: 256 x 256 tiles, cluster of two
// CTAs; A and B tensor maps both with boxes of 128 rows; needs
// GroupRows::mt2_prefix in grouped mode.  n_total must be a multiple of 128
// (SwiGLU) or 256 (down).
cudaError_t launch_swiglu_tc_pair(const TcGemmArgs& a, cudaStream_t stream);
cudaError_t launch_down_tc_pair(const TcGemmArgs& a, cudaStream_t stream);
int tc_n_granule(bool swiglu, int bn);  // output columns per tile
// 0 when n_total is not a multiple of the smaller granule.
int tc_pick_bn(bool swiglu, int n_total, int64_t mtiles_est, int num_sms);

// ---- combine (combine.cu) -------------------------------------------------
// out[t] = sum_{j<k_t} alpha[t,j] * y[row_of[t,j]] (+ y_shared[t]) (+ resid[t]).
cudaError_t launch_combine(int dtype, const void* y, const void* y_shared,
                           const void* resid, const int32_t* row_of, const float* alpha,
                           const int32_t* k, int T, int d, int k_max,
                           int cap_rows, void* out, uint32_t* err, int num_sms,
                           cudaStream_t stream);

}  // namespace rx
