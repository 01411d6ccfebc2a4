// reflex_abi.cu — the C ABI of include/reflex.h: argument checks, workspace
// carving, tensor-map construction and the launch sequence of one
// allocation call and one MoE-layer forward.  No allocation, no host sync
// (except the explicit status readers).
#include <cudaTypedefs.h>

#include <cmath>
#include <cstring>
#include <mutex>

#include "common.cuh"
#include "internal.h"
#include "reflex.h"

static_assert(sizeof(reflex_alloc_params) == 64, "reflex_alloc_params layout (ABI 113)");

namespace {

using rx::WsHeader;

constexpr size_t kAlign = 256;
// gate/up weight bytes handed to the L2 while the router scores run
constexpr uint64_t kRouterL2Prefetch = 64ull << 20;
// tokens from which layers with up to 64 experts screen their router scores
constexpr int32_t kBatchScreenMinTokens = 8192;      // up to 64 experts
// 65 to 256 experts: from 2048 tokens, where the per-token recheck starts
// (LLaDA2.0-mini shape: 2048 tokens 0.413 -> 0.394 ms, 4096 0.495 -> 0.478)
constexpr int32_t kBatchScreenMinTokensWide = 2048;
constexpr int32_t kBatchScreenMaxExperts = 256;
size_t up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

// Byte offsets of every workspace region (all 256-byte aligned).
struct Layout {
  size_t hdr, z, wnorm, tnorm, ids, alpha, blk_count, blk_mask, blk_off, counts, offsets,
      mt_prefix, mt2_prefix, perm, row_of, xperm, amid, ash, ysh, total;
  int64_t cap_rows;
  int nblk;
};

bool shapes_ok(int32_t dtype, int32_t T, int32_t d, int32_t E, int32_t inter,
               int32_t shared_inter, int32_t k_max) {
  if (dtype != REFLEX_DTYPE_F32 && dtype != REFLEX_DTYPE_BF16) return false;
  if (T < 0 || d <= 0 || d % 64 != 0 || E < 1 || E > 1024) return false;
  if (inter <= 0 || inter % 64 != 0) return false;
  if (shared_inter < 0 || shared_inter % 64 != 0) return false;
  if (k_max < 1 || k_max > 32) return false;
  if (static_cast<int64_t>(T) * k_max > (int64_t{1} << 30)) return false;
  return true;
}

Layout make_layout(int32_t dtype, int32_t T, int32_t d, int32_t E,
                   int32_t inter, int32_t shared_inter, int32_t k_max) {
  Layout L{};
  const size_t es = dtype == REFLEX_DTYPE_F32 ? 4 : 2;
  const int64_t cap = static_cast<int64_t>(T) * k_max;
  const int64_t nblk = rx::dispatch_blocks_alloc(T);
  size_t o = 0;
  auto take = [&](size_t bytes) {
    const size_t at = o;
    o += up(bytes);
    return at;
  };
  L.hdr = take(sizeof(WsHeader));
  // bf16: room for the screen GEMM's split-K slices of the scores
  const int64_t zrows = dtype == REFLEX_DTYPE_F32 ? T : rx::screen_z_rows(T, E, d);
  L.z = take(static_cast<size_t>(zrows) * E * 4);
  L.wnorm = take(static_cast<size_t>(E) * 4);
  L.tnorm = take(static_cast<size_t>(T) * 4);  // the batched screen's token sums of squares
  L.ids = take(cap * 4);
  L.alpha = take(cap * 4);
  L.blk_count = take(static_cast<size_t>(nblk) * E * 4);
  L.blk_mask = take(static_cast<size_t>(rx::dispatch_mask_words_alloc(T)) * E * 4);
  L.blk_off = take(static_cast<size_t>(nblk) * E * 4);
  L.counts = take(static_cast<size_t>(E) * 4);
  L.offsets = take(static_cast<size_t>(E + 1) * 4);
  L.mt_prefix = take(static_cast<size_t>(E + 1) * 4);
  L.mt2_prefix = take(static_cast<size_t>(E + 1) * 4);
  L.perm = take(cap * 4);
  L.row_of = take(cap * 4);
  L.xperm = take(cap * d * es);  // later reused for the expert outputs y
  L.amid = take(cap * inter * es);
  L.ash = shared_inter ? take(static_cast<size_t>(T) * shared_inter * es) : 0;
  L.ysh = shared_inter ? take(static_cast<size_t>(T) * d * es) : 0;
  L.total = o;
  L.cap_rows = cap;
  L.nblk = nblk;
  return L;
}

int num_sms_current() {
  static int cached[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 148;
  if (dev >= 0 && dev < 64 && cached[dev] > 0) return cached[dev];
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
    n = 148;
  if (dev >= 0 && dev < 64) cached[dev] = n;
  return n;
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                         cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// 2-D bf16 map over a row-major [rows, cols] matrix; box = 64 columns (128
// bytes, one swizzle row) x box_rows rows, 128-byte swizzle, zero fill.
bool make_map(CUtensorMap* m, const void* base, int64_t rows, int64_t cols,
              int box_rows) {
  auto fn = encode_fn();
  if (fn == nullptr) return false;
  if ((reinterpret_cast<uintptr_t>(base) & 15) != 0) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols) * 2};
  cuuint32_t box[2] = {64, static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base),
                  dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// Gate/up weights [groups][2][inter][K] as a 3D map {K, inter, 2 groups}:
// one box {64, box_rows, 2} holds a tile's gate rows and the matching up rows.
bool make_map_gate_up(CUtensorMap* m, const void* base, int64_t groups, int64_t inter,
                      int64_t cols, int box_rows) {
  auto fn = encode_fn();
  if (fn == nullptr) return false;
  if ((reinterpret_cast<uintptr_t>(base) & 15) != 0) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(inter),
                        static_cast<cuuint64_t>(2 * groups)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(cols) * 2,
                           static_cast<cuuint64_t>(inter) * static_cast<cuuint64_t>(cols) * 2};
  cuuint32_t box[3] = {64, static_cast<cuuint32_t>(box_rows), 2};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base),
                  dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

int map_err_bits(uint32_t bits) {
  if (bits == 0) return REFLEX_OK;
  if (bits & rx::kErrTimeout) return REFLEX_ETIMEOUT;
  if (bits & rx::kErrKRange) return REFLEX_EKRANGE;
  if (bits & rx::kErrCapacity) return REFLEX_ECAPACITY;
  return REFLEX_EINVAL;
}

#define RX_CUDA(x)                                  \
  do {                                              \
    if ((x) != cudaSuccess) return REFLEX_ECUDA;    \
  } while (0)

bool score_rule(const reflex_alloc_params* p) {
  return p->count_rule == REFLEX_RULE_TOP_P || p->count_rule == REFLEX_RULE_EXPERT_THRESHOLD;
}

// Argument checks of the allocation (reflex_allocate, reflex_step).  The
// score rules read no refinement state: only the counts' output is needed.
int check_alloc(const float* c1, const float* c2, const uint8_t* hl, const uint8_t* m,
                const int32_t* bid, const int32_t* so, const int32_t* act, int32_t T,
                int32_t B, const reflex_alloc_params* p, const int32_t* k_out) {
  if (p == nullptr || T < 0) return REFLEX_EINVAL;
  if (p->k_min < 1 || p->k_min > p->k_max || p->k_base < 1 ||
      p->delta_role < 0 || p->delta_cur < 0)
    return REFLEX_EINVAL;
  if (!(p->q > 0.0f && p->q <= 0.5f) || !(p->w_cf > 0.0f) || !(p->tau > 0.0f))
    return REFLEX_EINVAL;
  if (p->signal < REFLEX_SIGNAL_FPS || p->signal > REFLEX_SIGNAL_UNCERTAINTY ||
      (p->role_shuffle != 0 && p->role_shuffle != 1))
    return REFLEX_EINVAL;
  if (p->count_rule != REFLEX_RULE_REFLEX && !score_rule(p)) return REFLEX_EINVAL;
  if (score_rule(p)) {
    if (!std::isfinite(p->rule_threshold)) return REFLEX_EINVAL;
    if (T > 0 && k_out == nullptr) return REFLEX_EINVAL;
    return REFLEX_OK;
  }
  if (B < 1) return REFLEX_EINVAL;
  if (T > 0 && (c1 == nullptr || c2 == nullptr || hl == nullptr || m == nullptr ||
                bid == nullptr || k_out == nullptr))
    return REFLEX_EINVAL;
  if (so == nullptr || act == nullptr) return REFLEX_EINVAL;
  return REFLEX_OK;
}

// One allocation to run inside reflex_step.
struct AllocCall {
  const float* c1;
  const float* c2;
  const uint8_t* hl;
  const uint8_t* m;
  const int32_t* bid;
  const int32_t* so;
  const int32_t* act;
  int32_t B;
  rx::AllocArgs a;
  int32_t* k_out;
  unsigned long long* k_sum;
  uint32_t* err;
};

rx::AllocArgs alloc_args(const reflex_alloc_params* p) {
  return rx::AllocArgs{p->k_min, p->k_base,  p->k_max, p->delta_role, p->delta_cur,
                       p->q,     p->theta,   p->w_cf,  p->v_ref,      p->tau,
                       p->signal, p->role_shuffle, p->shuffle_seed, p->count_rule,
                       p->rule_threshold};
}

// The error word and the pair sum are stored outright by a single-sequence
// count kernel; with several sequences each CTA adds its share to cleared
// words, and so does every warp of the score rules' selection.
cudaError_t clear_alloc_outputs(const AllocCall& c, cudaStream_t s) {
  if (c.B <= 1 && c.a.count_rule == REFLEX_RULE_REFLEX) return cudaSuccess;
  if (c.err) {
    const cudaError_t e = cudaMemsetAsync(c.err, 0, sizeof(int32_t), s);
    if (e != cudaSuccess) return e;
  }
  if (c.k_sum) return cudaMemsetAsync(c.k_sum, 0, sizeof(int64_t), s);
  return cudaSuccess;
}

cudaError_t launch_alloc(const AllocCall& c, int32_t T, cudaStream_t s, bool alongside) {
  if (c.a.count_rule != REFLEX_RULE_REFLEX) return cudaSuccess;  // counts in the selection
  return rx::launch_budget(c.c1, c.c2, c.hl, c.m, c.bid, c.so, c.act, T, c.B, c.a, c.k_out,
                           c.k_sum, c.err, s, alongside);
}

}  // namespace

extern "C" {

int reflex_abi_version(void) { return 114; }

const char* reflex_status_string(int s) {
  switch (s) {
    case REFLEX_OK: return "ok";
    case REFLEX_EINVAL: return "invalid argument";
    case REFLEX_EKRANGE: return "expert count out of range";
    case REFLEX_EWORKSPACE: return "workspace missing or too small";
    case REFLEX_ECUDA: return "CUDA error";
    case REFLEX_ETIMEOUT: return "bounded device wait expired";
    case REFLEX_EUNSUPPORTED: return "shape not supported by the selected path";
    case REFLEX_ECAPACITY: return "too many active-block tokens in a sequence";
    default: return "unknown status";
  }
}

void reflex_default_params(reflex_alloc_params* p) {
  if (p == nullptr) return;
  p->k_min = 2;
  p->k_base = 8;
  p->k_max = 12;
  p->delta_role = 4;
  p->delta_cur = 2;
  p->q = 0.25f;
  p->theta = 0.9f;
  p->w_cf = 0.30f;
  p->v_ref = 0.01f;
  p->tau = 0.05f;
  p->signal = REFLEX_SIGNAL_FPS;
  p->role_shuffle = 0;
  p->shuffle_seed = 0;
  p->count_rule = REFLEX_RULE_REFLEX;
  p->rule_threshold = 0.0f;
}

int reflex_allocate(const float* router_scores, const float* conf_prev1,
                    const float* conf_prev2, const uint8_t* hist_len,
                    const uint8_t* masked, const int32_t* block_id,
                    const int32_t* seq_offsets, const int32_t* active_block,
                    int32_t T, int32_t B, int32_t E,
                    const reflex_alloc_params* p, int32_t* k_out,
                    int64_t* k_sum_out, int32_t* dev_status, void* stream) {
  const int chk = check_alloc(conf_prev1, conf_prev2, hist_len, masked, block_id,
                              seq_offsets, active_block, T, B, p, k_out);
  if (chk != REFLEX_OK) return chk;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (score_rule(p)) {
    // the counts of the threshold-based rules come from the router scores
    if (E < 1 || E > 1024 || (T > 0 && router_scores == nullptr)) return REFLEX_EINVAL;
    if (dev_status != nullptr) RX_CUDA(cudaMemsetAsync(dev_status, 0, sizeof(int32_t), s));
    if (k_sum_out != nullptr) RX_CUDA(cudaMemsetAsync(k_sum_out, 0, sizeof(int64_t), s));
    RX_CUDA(rx::launch_router_select_rule(router_scores, T, E, p->k_max, p->k_min,
                                          p->count_rule, p->rule_threshold, 1, true, k_out,
                                          reinterpret_cast<unsigned long long*>(k_sum_out),
                                          nullptr, nullptr, s));
    return REFLEX_OK;
  }
  const AllocCall c{conf_prev1, conf_prev2, hist_len, masked, block_id, seq_offsets,
                    active_block, B, alloc_args(p), k_out,
                    reinterpret_cast<unsigned long long*>(k_sum_out),
                    reinterpret_cast<uint32_t*>(dev_status)};
  RX_CUDA(clear_alloc_outputs(c, s));
  RX_CUDA(launch_alloc(c, T, s, false));
  return REFLEX_OK;
}

int reflex_update_state(const float* conf_new, float* conf_prev1, float* conf_prev2,
                        uint8_t* hist_len, uint8_t* masked, const int32_t* block_id,
                        const int32_t* seq_offsets, int32_t* active_block,
                        const int32_t* num_blocks, int32_t T, int32_t B,
                        float theta_commit, int32_t* committed_out,
                        int32_t* dev_status, void* stream) {
  if (T < 0 || B < 1 || !std::isfinite(theta_commit)) return REFLEX_EINVAL;
  if (seq_offsets == nullptr || active_block == nullptr || num_blocks == nullptr)
    return REFLEX_EINVAL;
  if (T > 0 && (conf_new == nullptr || conf_prev1 == nullptr || conf_prev2 == nullptr ||
                hist_len == nullptr || masked == nullptr || block_id == nullptr))
    return REFLEX_EINVAL;
  RX_CUDA(rx::launch_update_state(conf_new, conf_prev1, conf_prev2, hist_len, masked,
                                  block_id, seq_offsets, active_block, num_blocks, T, B,
                                  theta_commit, committed_out,
                                  reinterpret_cast<uint32_t*>(dev_status),
                                  static_cast<cudaStream_t>(stream)));
  return REFLEX_OK;
}

size_t reflex_moe_workspace_size(int32_t dtype, int32_t T, int32_t d,
                                 int32_t E, int32_t inter,
                                 int32_t shared_inter, int32_t k_max) {
  if (!shapes_ok(dtype, T, d, E, inter, shared_inter, k_max)) return 0;
  return make_layout(dtype, T, d, E, inter, shared_inter, k_max).total;
}

// The forward; with `ac`, the allocation of its counts too (k = ac->k_out):
// cleared outputs first, then the count kernel right behind the router
// scores, which it does not read, so the two run side by side.
static int forward_impl(int32_t dtype, const void* hidden, const void* w_router,
                        const void* w_gate_up, const void* w_down,
                        const void* shared_gate_up, const void* shared_down,
                        int32_t shared_inter, const int32_t* k, int32_t T,
                        int32_t d, int32_t E, int32_t inter, int32_t k_max,
                        uint32_t flags, void* workspace, size_t ws_bytes,
                        void* out, reflex_route_record* rec, void* stream,
                        const AllocCall* ac) {
  if (!shapes_ok(dtype, T, d, E, inter, shared_inter, k_max)) return REFLEX_EINVAL;
  if (shared_inter > 0 && (shared_gate_up == nullptr || shared_down == nullptr))
    return REFLEX_EINVAL;
  const Layout L = make_layout(dtype, T, d, E, inter, shared_inter, k_max);
  if (workspace == nullptr || ws_bytes < L.total) return REFLEX_EWORKSPACE;
  if ((reinterpret_cast<uintptr_t>(workspace) & (kAlign - 1)) != 0)
    return REFLEX_EWORKSPACE;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  WsHeader* hdr = reinterpret_cast<WsHeader*>(ws + L.hdr);
  int32_t* totals = &hdr->total_pairs;
  uint32_t* err = &hdr->err;
  auto I32 = [&](size_t off) { return reinterpret_cast<int32_t*>(ws + off); };
  if (rec != nullptr) {
    rec->ids = I32(L.ids);
    rec->alpha = reinterpret_cast<float*>(ws + L.alpha);
    rec->counts = I32(L.counts);
    rec->offsets = I32(L.offsets);
    rec->perm = I32(L.perm);
    rec->row_of = I32(L.row_of);
    rec->totals = totals;
    rec->scores = reinterpret_cast<float*>(ws + L.z);
  }
  if (T == 0) {
    // no kernel of the layer runs: the header (error word, totals) still
    // describes this call
    cudaStream_t s0 = static_cast<cudaStream_t>(stream);
    RX_CUDA(cudaMemsetAsync(hdr, 0, sizeof(WsHeader), s0));
    if (ac != nullptr) {
      RX_CUDA(clear_alloc_outputs(*ac, s0));
      RX_CUDA(launch_alloc(*ac, 0, s0, false));
    }
    return REFLEX_OK;
  }
  if (hidden == nullptr || w_router == nullptr || w_gate_up == nullptr ||
      w_down == nullptr || k == nullptr || out == nullptr)
    return REFLEX_EINVAL;

  const bool simt = dtype == REFLEX_DTYPE_F32 || (flags & REFLEX_FLAG_SIMT_EXPERTS);
  // tile widths of the tcgen05 GEMMs: the m-tile count is only known on the
  // device, so the choice uses the expected count for pairs spread over
  // every expert (one partial tile per expert plus T k_max / 2 rows)
  const int sms_h = num_sms_current();
  const int64_t mt_est = E + (static_cast<int64_t>(T) * k_max / 2 + 127) / 128;
  const int64_t mt_dense = (T + 127) / 128;
  const int bn_up = rx::tc_pick_bn(true, inter, mt_est, sms_h);
  const int bn_dn = rx::tc_pick_bn(false, d, mt_est, sms_h);
  const int bn_sup = shared_inter ? rx::tc_pick_bn(true, shared_inter, mt_dense, sms_h) : 128;
  const int bn_sdn = shared_inter ? rx::tc_pick_bn(false, d, mt_dense, sms_h) : 128;
  // CTA-pair (2-SM) GEMMs once the groups are expected to outgrow one
  // 128-row tile: a 256-row pair tile covers a group of a few hundred rows in
  // one pass (the 1-SM kernel would stream every weight tile once per m-tile,
  // the last one mostly padding) and each SM streams half of the weights
  // (LLaDA2.0-mini layer, about 160 rows per expert: 0.820 -> 0.749 ms)
  const int64_t rows_per_group_est = static_cast<int64_t>(T) * k_max / 2 / E;
  const bool pair_routed = rows_per_group_est >= 128 && inter % 128 == 0 && d % 256 == 0;
  // fused dispatch (opt-in): the CTA-pair gate/up GEMM gathers its rows from
  // hidden through perm, and the dispatch only places the pairs
  const bool gemm_gathers = !simt && pair_routed && (flags & REFLEX_FLAG_GATHER_IN_GEMM);
  if (!simt) {
    if (bn_up == 0 || bn_dn == 0 || bn_sup == 0 || bn_sdn == 0) return REFLEX_EUNSUPPORTED;
    if (encode_fn() == nullptr) return REFLEX_ECUDA;
  }
  constexpr uint32_t kAllStages = REFLEX_STAGE_ROUTE | REFLEX_STAGE_DISPATCH |
                                  REFLEX_STAGE_EXPERT_UP | REFLEX_STAGE_EXPERT_DOWN |
                                  REFLEX_STAGE_COMBINE;
  uint32_t stages = flags & kAllStages;
  if (stages == 0) stages = kAllStages;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int sms = sms_h;
  const int cap = static_cast<int>(L.cap_rows);
  float* z = reinterpret_cast<float*>(ws + L.z);
  float* alpha = reinterpret_cast<float*>(ws + L.alpha);
  void* xperm = ws + L.xperm;  // gathered rows, then expert outputs y
  void* amid = ws + L.amid;
  void* ash = shared_inter ? ws + L.ash : nullptr;
  void* ysh = shared_inter ? ws + L.ysh : nullptr;

  if (ac != nullptr) RX_CUDA(clear_alloc_outputs(*ac, s));
  // bf16 with renormalised weights, many experts and many scores: tensor-
  // core scores screen the experts and only those that could be selected get
  // the canonical chain (router.cu).  The recheck costs about as much per
  // chain as 40 chains of the dense score kernels and has a latency floor, so
  // it pays from 128 experts and 2048 x 256 scores on (LLaDA2.0-mini layer:
  // routing 213 -> 113 us at 8192 tokens, layer 4.90 -> 4.35 ms at 65536;
  // below 2048 tokens, and with 64 experts at every size, the dense kernels
  // are faster).
  // the score rules' counts need every score from the chain: no screen
  const bool rule = ac != nullptr && ac->a.count_rule != REFLEX_RULE_REFLEX;
  const bool screen = dtype == REFLEX_DTYPE_BF16 && (flags & REFLEX_FLAG_RENORM_TOPK) &&
                      !(flags & REFLEX_FLAG_EXACT_SCORES) && d % 128 == 0 && E >= 128 &&
                      static_cast<int64_t>(T) * E >= 2048 * 256 && !rule;
  // the same screen batched, for up to 256 experts and many tokens: the
  // score GEMM also sums the squares of the token rows, and the recheck
  // streams a block of token rows and every expert row through shared
  // memory, one chain per candidate pair (router.cu); it takes precedence
  // over the per-token recheck (LLaDA2.0-mini layer 0.573 -> 0.546 ms)
  const bool batch_screen = dtype == REFLEX_DTYPE_BF16 && (flags & REFLEX_FLAG_RENORM_TOPK) &&
                            !(flags & REFLEX_FLAG_EXACT_SCORES) && !rule &&
                            E <= kBatchScreenMaxExperts && d % 64 == 0 &&
                            T >= (E <= 64 ? kBatchScreenMinTokens : kBatchScreenMinTokensWide);
  if ((stages & REFLEX_STAGE_ROUTE) && batch_screen) {
    CUtensorMap mh, mw, mhb, mwb;
    const int sbn = E <= 64 ? 64 : 128;  // score tile width
    if (!make_map(&mh, hidden, T, d, rx::kTileM) || !make_map(&mw, w_router, E, d, sbn) ||
        !make_map(&mhb, hidden, T, d, rx::screen_batch_token_rows(E)) ||
        !make_map(&mwb, w_router, E, d, rx::screen_batch_expert_rows(E)))
      return REFLEX_ECUDA;
    float* nw = reinterpret_cast<float*>(ws + L.wnorm);
    float* hss = reinterpret_cast<float*>(ws + L.tnorm);
    RX_CUDA(rx::launch_router_wnorm(static_cast<const __nv_bfloat16*>(w_router), E, d, nw,
                                    reinterpret_cast<uint32_t*>(hdr),
                                    static_cast<int>(sizeof(WsHeader) / 4), s));
    rx::GroupRows rows{nullptr, nullptr, nullptr, nullptr, 1, T, T};
    rx::TcGemmArgs sa{&mh, &mw, d, E, 0, 0, rows, nullptr, E, err, sms};
    RX_CUDA(rx::launch_scores_tc(sa, sbn, 1, z, static_cast<int64_t>(T) * E, E, true, s, hss));
    if (ac != nullptr) RX_CUDA(launch_alloc(*ac, T, s, true));
    RX_CUDA(rx::launch_router_screen_batch(&mhb, &mwb, z, hss, nw, k, T, E, d, k_max,
                                           I32(L.ids), alpha, err, s));
  } else if ((stages & REFLEX_STAGE_ROUTE) && screen) {
    const int bn = rx::screen_bn(E), ks = rx::screen_splits(T, E, d);
    CUtensorMap mh, mw;
    if (!make_map(&mh, hidden, T, d, rx::kTileM) || !make_map(&mw, w_router, E, d, bn))
      return REFLEX_ECUDA;
    float* nw = reinterpret_cast<float*>(ws + L.wnorm);
    const int64_t zs = static_cast<int64_t>(T) * E;
    // the first kernel clears the header (error word, totals); the score GEMM
    // reads and writes nothing it touches, so it runs beside it, and so does
    // the count kernel of reflex_step
    RX_CUDA(rx::launch_router_wnorm(static_cast<const __nv_bfloat16*>(w_router), E, d, nw,
                                    reinterpret_cast<uint32_t*>(hdr),
                                    static_cast<int>(sizeof(WsHeader) / 4), s));
    rx::GroupRows rows{nullptr, nullptr, nullptr, nullptr, 1, T, T};
    rx::TcGemmArgs sa{&mh, &mw, d, E, 0, 0, rows, nullptr, E, err, sms};
    RX_CUDA(rx::launch_scores_tc(sa, bn, ks, z, zs, E, true, s));
    if (ac != nullptr) RX_CUDA(launch_alloc(*ac, T, s, true));
    RX_CUDA(rx::launch_router_screen_select(
        static_cast<const __nv_bfloat16*>(hidden), static_cast<const __nv_bfloat16*>(w_router),
        z, ks, zs, nw, k, T, E, d, k_max, I32(L.ids), alpha, err, s));
  } else if (stages & REFLEX_STAGE_ROUTE) {
    // the router's first CTA clears the header (error word, totals): no
    // kernel before the router reads it
    // the first experts' gate/up weights are handed to the L2 while the
    // scores run (the grouped GEMM walks the experts in order; LLaDA-MoE
    // layer step -2 us with 64 MB)
    rx::L2Prefetch pf;
    if (stages & REFLEX_STAGE_EXPERT_UP) {
      const uint64_t wbytes =
          static_cast<uint64_t>(E) * 2 * inter * d * (dtype == REFLEX_DTYPE_F32 ? 4 : 2);
      pf.base = w_gate_up;
      pf.bytes = (wbytes < kRouterL2Prefetch ? wbytes : kRouterL2Prefetch) & ~uint64_t{4095};
    }
    RX_CUDA(rx::launch_router_logits(dtype, hidden, w_router, T, d, E, z,
                                     reinterpret_cast<uint32_t*>(hdr),
                                     static_cast<int>(sizeof(WsHeader) / 4), err, sms, s, pf));
    if (rule) {
      // k = ac->k_out: the selection writes the counts it derives
      RX_CUDA(rx::launch_router_select_rule(z, T, E, ac->a.k_max < k_max ? ac->a.k_max : k_max,
                                            ac->a.k_min,
                                            ac->a.count_rule, ac->a.rule_threshold, k_max,
                                            (flags & REFLEX_FLAG_RENORM_TOPK) != 0,
                                            ac->k_out, ac->k_sum, I32(L.ids), alpha, s));
    } else {
      if (ac != nullptr) RX_CUDA(launch_alloc(*ac, T, s, true));
      RX_CUDA(rx::launch_router_select(z, k, T, E, k_max,
                                       (flags & REFLEX_FLAG_RENORM_TOPK) != 0,
                                       I32(L.ids), alpha, err, s));
    }
  } else if (ac != nullptr) {
    RX_CUDA(launch_alloc(*ac, T, s, false));
  }
  if (stages & REFLEX_STAGE_DISPATCH) {
    rx::DispatchBufs b{I32(L.blk_count), I32(L.blk_off),   I32(L.counts),
                       I32(L.offsets),   I32(L.mt_prefix), I32(L.mt2_prefix),
                       I32(L.perm),      I32(L.row_of),    totals,
                       err,              reinterpret_cast<uint32_t*>(ws + L.blk_mask)};
    RX_CUDA(rx::launch_dispatch_gather(dtype, hidden, I32(L.ids), k, T, E, k_max, cap, d, b,
                                       gemm_gathers ? nullptr : xperm, sms, s));
  }
  const bool up = (stages & REFLEX_STAGE_EXPERT_UP) != 0;
  const bool down = (stages & REFLEX_STAGE_EXPERT_DOWN) != 0;
  if (up || down) {
    rx::GroupRows grouped{I32(L.offsets), I32(L.mt_prefix), I32(L.mt2_prefix), totals,
                          E, 0, cap};
    rx::GroupRows dense{nullptr, nullptr, nullptr, nullptr, 1, T, T};
    if (simt) {
      if (up) {
        RX_CUDA(rx::launch_swiglu_simt(dtype, xperm, w_gate_up, d, inter, grouped, amid, err, s));
        if (shared_inter)
          RX_CUDA(rx::launch_swiglu_simt(dtype, hidden, shared_gate_up, d, shared_inter, dense, ash, err, s));
      }
      if (down) {
        RX_CUDA(rx::launch_down_simt(dtype, amid, w_down, d, inter, grouped, xperm, err, s));
        if (shared_inter)
          RX_CUDA(rx::launch_down_simt(dtype, ash, shared_down, d, shared_inter, dense, ysh, err, s));
      }
    } else {
      CUtensorMap ma1, mb1, ma2, mb2;
      if (!(gemm_gathers ? make_map(&ma1, hidden, T, d, 1)
                         : make_map(&ma1, xperm, cap, d, rx::kTileM)) ||
          !(pair_routed ? make_map(&mb1, w_gate_up, static_cast<int64_t>(E) * 2 * inter, d, 128)
                        : make_map_gate_up(&mb1, w_gate_up, E, inter, d,
                                           rx::tc_b_box_rows(true, bn_up))) ||
          !make_map(&ma2, amid, cap, inter, rx::kTileM) ||
          !make_map(&mb2, w_down, static_cast<int64_t>(E) * d, inter,
                    pair_routed ? 128 : rx::tc_b_box_rows(false, bn_dn)))
        return REFLEX_ECUDA;
      rx::TcGemmArgs g1{&ma1, &mb1, d, inter, 2 * inter, inter, grouped, amid, inter, err, sms,
                        !pair_routed};
      if (gemm_gathers) {
        g1.gather_perm = I32(L.perm);
        g1.gather_kmax = k_max;
        g1.gather_tokens = T;
      }
      rx::TcGemmArgs g2{&ma2, &mb2, inter, d, d, 0, grouped, xperm, d, err, sms};
      // output maps of the CTA-pair GEMMs (whole 32-row chunks by TMA store)
      CUtensorMap mo1, mo2;
      if (pair_routed) {
        if (!make_map(&mo1, amid, cap, inter, 32) || !make_map(&mo2, xperm, cap, d, 32))
          return REFLEX_ECUDA;
        g1.map_out = &mo1;
        g2.map_out = &mo2;
      }
      // the dense shared expert on CTA pairs once it has enough rows: a 256 x
      // 256 pair tile moves a quarter of the operand bytes per output that a
      // 128 x 128 tile of the 1-SM kernel moves from L2 (LLaDA2.0-mini layer
      // 0.750 -> 0.736 ms; at 1024 tokens the 1-SM tiles stay 6 us faster)
      const bool pair_shared =
          shared_inter > 0 && T >= 2048 && shared_inter % 128 == 0 && d % 256 == 0;
      CUtensorMap sa1, sb1, sa2, sb2;
      if (shared_inter &&
          (!make_map(&sa1, hidden, T, d, rx::kTileM) ||
           !(pair_shared
                 ? make_map(&sb1, shared_gate_up, 2 * static_cast<int64_t>(shared_inter), d, 128)
                 : make_map_gate_up(&sb1, shared_gate_up, 1, shared_inter, d,
                                    rx::tc_b_box_rows(true, bn_sup))) ||
           !make_map(&sa2, ash, T, shared_inter, rx::kTileM) ||
           !make_map(&sb2, shared_down, d, shared_inter,
                     pair_shared ? 128 : rx::tc_b_box_rows(false, bn_sdn))))
        return REFLEX_ECUDA;
      rx::TcGemmArgs h1{&sa1, &sb1, d, shared_inter, 2 * shared_inter, shared_inter,
                        dense, ash, shared_inter, err, sms, !pair_shared};
      rx::TcGemmArgs h2{&sa2, &sb2, shared_inter, d, d, 0, dense, ysh, d, err, sms};
      CUtensorMap so1, so2;
      if (pair_shared) {
        if (!make_map(&so1, ash, T, shared_inter, 32) || !make_map(&so2, ysh, T, d, 32))
          return REFLEX_ECUDA;
        h1.map_out = &so1;
        h2.map_out = &so2;
      }
      if (up) {
        if (pair_routed)
          RX_CUDA(rx::launch_swiglu_tc_pair(g1, s));
        else
          RX_CUDA(rx::launch_swiglu_tc(g1, bn_up, s));
        if (shared_inter) {
          if (pair_shared)
            RX_CUDA(rx::launch_swiglu_tc_pair(h1, s));
          else
            RX_CUDA(rx::launch_swiglu_tc(h1, bn_sup, s));
        }
      }
      if (down) {
        if (pair_routed)
          RX_CUDA(rx::launch_down_tc_pair(g2, s));
        else
          RX_CUDA(rx::launch_down_tc(g2, bn_dn, s));
        if (shared_inter) {
          if (pair_shared)
            RX_CUDA(rx::launch_down_tc_pair(h2, s));
          else
            RX_CUDA(rx::launch_down_tc(h2, bn_sdn, s));
        }
      }
    }
  }
  if (stages & REFLEX_STAGE_COMBINE) {
    const void* resid = (flags & REFLEX_FLAG_RESIDUAL) ? hidden : nullptr;
    RX_CUDA(rx::launch_combine(dtype, xperm, ysh, resid, I32(L.row_of), alpha, k, T, d,
                               k_max, cap, out, err, sms, s));
  }
  return REFLEX_OK;
}

int reflex_moe_forward(int32_t dtype, const void* hidden, const void* w_router,
                       const void* w_gate_up, const void* w_down,
                       const void* shared_gate_up, const void* shared_down,
                       int32_t shared_inter, const int32_t* k, int32_t T,
                       int32_t d, int32_t E, int32_t inter, int32_t k_max,
                       uint32_t flags, void* workspace, size_t ws_bytes,
                       void* out, reflex_route_record* rec, void* stream) {
  return forward_impl(dtype, hidden, w_router, w_gate_up, w_down, shared_gate_up,
                      shared_down, shared_inter, k, T, d, E, inter, k_max, flags,
                      workspace, ws_bytes, out, rec, stream, nullptr);
}

int reflex_step(const float* conf_prev1, const float* conf_prev2, const uint8_t* hist_len,
                const uint8_t* masked, const int32_t* block_id, const int32_t* seq_offsets,
                const int32_t* active_block, int32_t B, const reflex_alloc_params* p,
                int32_t* k_out, int64_t* k_sum_out, int32_t* alloc_status,
                int32_t dtype, const void* hidden, const void* w_router,
                const void* w_gate_up, const void* w_down, const void* shared_gate_up,
                const void* shared_down, int32_t shared_inter, int32_t T, int32_t d,
                int32_t E, int32_t inter, int32_t k_max, uint32_t flags, void* workspace,
                size_t ws_bytes, void* out, reflex_route_record* rec, void* stream) {
  const int chk = check_alloc(conf_prev1, conf_prev2, hist_len, masked, block_id,
                              seq_offsets, active_block, T, B, p, k_out);
  if (chk != REFLEX_OK) return chk;
  if (T > 0 && k_out == nullptr) return REFLEX_EINVAL;
  // with a score rule the counts come out of the ROUTE stage
  const uint32_t st_bits = flags & (REFLEX_STAGE_ROUTE | REFLEX_STAGE_DISPATCH |
                                    REFLEX_STAGE_EXPERT_UP | REFLEX_STAGE_EXPERT_DOWN |
                                    REFLEX_STAGE_COMBINE);
  if (score_rule(p) && st_bits != 0 && !(st_bits & REFLEX_STAGE_ROUTE)) return REFLEX_EINVAL;
  const AllocCall c{conf_prev1, conf_prev2, hist_len, masked, block_id, seq_offsets,
                    active_block, B, alloc_args(p), k_out,
                    reinterpret_cast<unsigned long long*>(k_sum_out),
                    reinterpret_cast<uint32_t*>(alloc_status)};
  return forward_impl(dtype, hidden, w_router, w_gate_up, w_down, shared_gate_up,
                      shared_down, shared_inter, k_out, T, d, E, inter, k_max, flags,
                      workspace, ws_bytes, out, rec, stream, &c);
}

int reflex_read_status(const int32_t* dev_status, void* stream) {
  if (dev_status == nullptr) return REFLEX_EINVAL;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  uint32_t bits = 0;
  RX_CUDA(cudaMemcpyAsync(&bits, dev_status, sizeof(bits), cudaMemcpyDeviceToHost, s));
  RX_CUDA(cudaStreamSynchronize(s));
  return map_err_bits(bits);
}

int reflex_moe_status(const void* workspace, void* stream) {
  if (workspace == nullptr) return REFLEX_EINVAL;
  const WsHeader* hdr = static_cast<const WsHeader*>(workspace);
  return reflex_read_status(reinterpret_cast<const int32_t*>(&hdr->err), stream);
}

int reflex_selftest_wait_timeout(int32_t* dev_status, uint32_t limit_us,
                                 void* stream) {
  if (dev_status == nullptr || limit_us < 1 || limit_us > 100000) return REFLEX_EINVAL;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  RX_CUDA(cudaMemsetAsync(dev_status, 0, sizeof(int32_t), s));
  RX_CUDA(rx::launch_wait_selftest(reinterpret_cast<uint32_t*>(dev_status),
                                   static_cast<uint64_t>(limit_us) * 1000ull, s));
  return REFLEX_OK;
}

}  // extern "C"
