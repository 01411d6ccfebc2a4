/*
 * reflex.h — C ABI of the REFLEX per-forward MoE hot path on one GB300
 * (sm_103a).  Library: paper_2608_01784_gb300/_build/libreflex.so.
 *
 * REFLEX (arxiv 2608.01784) splits token-choice MoE inference into expert
 * ranking (left to the default router) and expert-count allocation.  This
 * library implements both halves of one denoising forward:
 *
 *   reflex_allocate     the allocation rule k = Pi(S_t, K^Sigma) of Eq. 3,
 *                       realised by Refinement-Role Budgeting (Sec. 4.2,
 *                       Eq. 5) and Frontier-Guided Expert Reallocation
 *                       (Sec. 4.3, Eq. 6-9), clipped to [K_min, K_max].
 *   reflex_moe_forward  the variable-count MoE layer of Eq. 2: router scores,
 *                       TopK(r_i, k_i), normalised router weights, SwiGLU
 *                       experts on the selected token-expert pairs, weighted
 *                       sum (plus an optional always-on shared expert).
 *
 * Conventions shared by every call
 *   - All array arguments are DEVICE pointers unless stated otherwise; the
 *     caller owns them.  The library never allocates or frees device memory
 *     and never synchronises the stream, except reflex_moe_status and
 *     reflex_read_status, which synchronise to read an error word.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy stream).  All
 *     work is enqueued asynchronously on it.
 *   - Row-major layouts.  Integer arrays are int32 unless stated.
 *   - Return value: a REFLEX_* status.  Host-side checks (null pointers,
 *     shapes, workspace size) return before anything is enqueued.  Checks
 *     that need device data (a count k_i out of range, too many active-block
 *     tokens) set bits in a device error word; read it with
 *     reflex_moe_status / reflex_read_status.
 */
#ifndef REFLEX_H
#define REFLEX_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ------------------------------------------------------- */
#define REFLEX_OK 0
#define REFLEX_EINVAL 1        /* null pointer, bad shape or parameter       */
#define REFLEX_EKRANGE 2       /* a count outside its allowed range          */
#define REFLEX_EWORKSPACE 3    /* workspace missing or smaller than needed   */
#define REFLEX_ECUDA 4         /* a CUDA runtime / launch error              */
#define REFLEX_ETIMEOUT 5      /* a bounded device wait expired              */
#define REFLEX_EUNSUPPORTED 6  /* shape not supported by the selected path   */
#define REFLEX_ECAPACITY 7     /* more active-block tokens than supported    */

/* ---- element types ------------------------------------------------------ */
#define REFLEX_DTYPE_F32 0     /* fp32 storage and fp32 arithmetic           */
#define REFLEX_DTYPE_BF16 1    /* bf16 storage, fp32 accumulation            */

/* ---- reflex_moe_forward flags ------------------------------------------ */
/* alpha renormalised over the selected experts (default reading of the
 * "normalized router weight" of Sec. 3.2); without it alpha is the softmax
 * over all E experts. */
#define REFLEX_FLAG_RENORM_TOPK 0x1u
/* bf16 only: run the expert GEMMs on the SIMT kernels instead of the
 * tcgen05/TMEM kernels (cross-checking; the fp32 path always uses SIMT). */
#define REFLEX_FLAG_SIMT_EXPERTS 0x2u
/* Residual connection for stacked layers: out = hidden + MoE(hidden), summed
 * in fp32 with the expert outputs and rounded once. */
#define REFLEX_FLAG_RESIDUAL 0x4u
/* bf16: compute every router score with the canonical fma chain.  Without
 * it (and with REFLEX_FLAG_RENORM_TOPK) the scores come from a tensor-core
 * GEMM and only the experts that could be selected are recomputed with the
 * chain: the selected experts, their weights and their scores are the same
 * bits either way (the screen's bound is stated with reflex_moe_forward);
 * only the record's other scores differ (tensor-core estimates). */
#define REFLEX_FLAG_EXACT_SCORES 0x8u
/* bf16 tcgen05 path, routed gate/up GEMM on CTA pairs (at least 128 rows
 * per expert expected: T * k_max / (2 E) >= 128, inter % 128 == 0, d % 256
 * == 0): the GEMM fetches its input rows from hidden itself with four-row
 * TMA gathers through the pair permutation, and DISPATCH only places the
 * pairs (no copy of the rows in pair order is written).  The outputs are the
 * same bits as without the flag.  Elsewhere the flag changes nothing.  The
 * fused dispatch is slower on GB300 (a four-row gather costs about four
 * times what a row of a tiled box does: the 32 x 1024-token LLaDA-MoE layer's
 * gate/up GEMM 0.84 -> 3.08 ms), so it is off by default.  With stage
 * selection the DISPATCH and EXPERT_UP calls must agree on the flag. */
#define REFLEX_FLAG_GATHER_IN_GEMM 0x10u
/* Stage selection.  No stage bit = all five stages in order.  Stages read
 * what the previous stages left in the same workspace; running a stage whose
 * predecessors did not run on that workspace gives unspecified values (every
 * index read from the workspace is range-checked on the device, so no
 * out-of-bounds access results).  hidden must hold the same values at the
 * DISPATCH and EXPERT_UP stages of one forward (the shared expert reads it
 * at EXPERT_UP, and so do the routed experts with REFLEX_FLAG_GATHER_IN_GEMM)
 * and, with REFLEX_FLAG_RESIDUAL, at COMBINE. */
#define REFLEX_STAGE_ROUTE 0x100u       /* router scores, TopK, alpha        */
#define REFLEX_STAGE_DISPATCH 0x200u    /* pair counts, offsets, permutation */
#define REFLEX_STAGE_EXPERT_UP 0x400u   /* gate/up GEMM + SwiGLU (+ shared)  */
#define REFLEX_STAGE_EXPERT_DOWN 0x800u /* down GEMM (+ shared)              */
#define REFLEX_STAGE_COMBINE 0x1000u    /* weighted sum back to token order  */

/* ---- allocation hyper-parameters (Sec. 4.2-4.3; defaults in Sec. 5.1) --- */
typedef struct {
    int32_t k_min;      /* lower clip bound of every count, >= 1            */
    int32_t k_base;     /* K_base of Eq. 5                                  */
    int32_t k_max;      /* upper clip bound, >= k_min                       */
    int32_t delta_role; /* delta_role of Eq. 5 (0 = no role prior)          */
    int32_t delta_cur;  /* delta_cur of Eq. 9 (0 = no reallocation)         */
    float q;            /* outer-group fraction of Eq. 9, in (0, 1/2]       */
    float theta;        /* commitment threshold of Eq. 6                    */
    float w_cf;         /* commitment-frontier width of Eq. 6 and the
                           velocity clip, > 0                               */
    float v_ref;        /* velocity reference of Eq. 7                      */
    float tau;          /* gate temperature of Eq. 6-7, > 0                 */
    int32_t signal;     /* rank key of the Eq. 9 groups: REFLEX_SIGNAL_*    */
    int32_t role_shuffle; /* 1: permute each sequence's final counts among
                           its positions (Role-Shuffled RRB, App. C); the
                           multiset and sum of the counts are unchanged.
                           Sequences longer than 4096 tokens are left as
                           they are and flag REFLEX_ECAPACITY.              */
    uint64_t shuffle_seed; /* seed of the shuffle's splitmix64 stream       */
    int32_t count_rule; /* where the counts come from: REFLEX_RULE_*        */
    float rule_threshold; /* p of REFLEX_RULE_TOP_P, or the router-weight
                           threshold of REFLEX_RULE_EXPERT_THRESHOLD      */
} reflex_alloc_params;

/* Count rules.  REFLEX_RULE_REFLEX (0, the default) is the allocation of
 * Sec. 4.2-4.3 above.  The other two are the threshold-based comparison
 * methods of App. B, which take each token's count from its router scores
 * z_t instead of its refinement state (the paper runs them with the count
 * bounds [1, 12], i.e. k_min = 1, k_max = 12):
 *   TOP_P             the smallest prefix of the router-ranked experts
 *                     (scores descending, lower index first on ties) whose
 *                     cumulative routing mass reaches rule_threshold;
 *   EXPERT_THRESHOLD  the number of experts whose routing mass exceeds
 *                     rule_threshold;
 * either clipped to [k_min, min(k_max, E)].  The routing mass is the
 * softmax of z_t over all E experts, and the decision is taken in fp32 in
 * this order, so that the counts are reproducible bit for bit:
 *   m = max_e z_e;  u_e = exp(z_e - m) (the library's Cody-Waite exp, the
 *   one of the FPS sigmoids);  S = the sum of the u_e, lane l of 32 adding
 *   u_l, u_{l+32}, ... in ascending order, then the 32 lane sums combined by
 *   s_l <- s_l + s_{l xor o} for o = 16, 8, 4, 2, 1;
 *   TOP_P: c_j = c_{j-1} + u_(j) over the ranks j = 1, 2, ... (c_0 = 0),
 *   k = the smallest j with c_j / S >= rule_threshold;
 *   EXPERT_THRESHOLD: k = #{e : u_e / S > rule_threshold}.
 * The score rules read every router score, so a forward that takes its
 * counts from them computes every score with the canonical chain (as with
 * REFLEX_FLAG_EXACT_SCORES). */
#define REFLEX_RULE_REFLEX 0
#define REFLEX_RULE_TOP_P 1
#define REFLEX_RULE_EXPERT_THRESHOLD 2

/* Rank keys for the FGER groups (Sec. 4.3; signal ablation of App. C).  The
 * top floor(q |J_h|) tokens by (key desc, position asc) gain delta_cur, the
 * bottom ones lose it.
 *   FPS          S = F * P (Eq. 8), the REFLEX default
 *   FRONTIER     F alone (Eq. 6)
 *   PROGRESS     P alone (Eq. 7; 1 with fewer than two observations)
 *   CONFIDENCE   c^{t-1}
 *   UNCERTAINTY  1 - c^{t-1} (fp32)
 * RRB Only and FGER Only (Sec. 5.3) are parameter settings: delta_cur = 0 and
 * delta_role = 0 respectively. */
#define REFLEX_SIGNAL_FPS 0
#define REFLEX_SIGNAL_FRONTIER 1
#define REFLEX_SIGNAL_PROGRESS 2
#define REFLEX_SIGNAL_CONFIDENCE 3
#define REFLEX_SIGNAL_UNCERTAINTY 4

/* Role shuffle.  Token i of a sequence gets the key
 *   key_i = high 32 bits of splitmix64 output number i + 1 for shuffle_seed
 * (splitmix64: state_n = seed + n * 0x9e3779b97f4a7c15, output = the
 * Stafford "mix13" finaliser of state_n, Steele, Lea and Flood 2014), i the
 * token's index in the batch; with r_i the rank of (key_i, i) in ascending
 * order within the sequence, token i receives the count the unshuffled
 * allocation gives to the sequence's r_i-th position. */

/* Fills the Sec. 5.1 defaults: k_base 8, delta_role 4, delta_cur 2, q 0.25,
 * theta 0.9, w_cf 0.30 (LLaDA-MoE; 0.25 for LLaDA2.0-mini), v_ref 0.01,
 * tau 0.05, the clip [k_min, k_max] = [2, 12], signal FPS, no shuffle,
 * count rule REFLEX (rule_threshold 0). */
void reflex_default_params(reflex_alloc_params* p);

/*
 * reflex_allocate — per-token expert counts k_i for one denoising forward
 * (Eq. 3 realised by Eq. 5 and Eq. 9, Sec. 4.2-4.3).
 *
 *   router_scores  [T, E] fp32.  REFLEX's rule does not read it (the router
 *                  only ranks experts, Sec. 3.3) and it may be NULL; the
 *                  score rules (p->count_rule TOP_P or EXPERT_THRESHOLD)
 *                  take the counts from it alone (E experts per row), and
 *                  then every state array below may be NULL.
 *   conf_prev1     [T] fp32  c_i^{t-1}, the latest confidence observation.
 *   conf_prev2     [T] fp32  c_i^{t-2}; read only where hist_len >= 2.
 *   hist_len       [T] u8    number of past observations (0, 1, >= 2).
 *   masked         [T] u8    1 = position is [MASK] (member of M_t).
 *   block_id       [T] int32 b(i): 0 for prompt positions, 1..Q for target
 *                            blocks.
 *   seq_offsets    [B+1]     token range of each sequence; seq_offsets[0] = 0,
 *                            seq_offsets[B] = T, non-decreasing.
 *   active_block   [B]       a_t of each sequence, >= 1.
 *   p              HOST pointer to the hyper-parameters.
 *   k_out          [T] int32 output counts, each in [k_min, k_max].
 *   k_sum_out      [1] int64 nullable: sum of k_out (the realised budget).
 *   dev_status     [1] int32 nullable device error word; cleared by this
 *                  call, then OR-ed with error bits (see reflex_read_status).
 * Tokens of the active block that are masked and have at least one
 * observation form J_h and are ranked by the Frontier-Progress Score (ties:
 * lower position first); at most 4096 such tokens per sequence (more sets
 * REFLEX_ECAPACITY in dev_status and leaves them at K_cur, clipped).
 * Host errors: REFLEX_EINVAL for null required pointers, T < 0, B < 1, or
 * parameters violating 1 <= k_min <= k_max, k_base >= 1, delta_* >= 0,
 * 0 < q <= 0.5, w_cf > 0, tau > 0, an unknown count_rule, or (score rules)
 * a missing router_scores, E outside [1, 1024] or a non-finite
 * rule_threshold.  Counts below k_min (or above k_max) produced by Eq. 5 /
 * Eq. 9 are clipped.
 */
int reflex_allocate(const float* router_scores, const float* conf_prev1,
                    const float* conf_prev2, const uint8_t* hist_len,
                    const uint8_t* masked, const int32_t* block_id,
                    const int32_t* seq_offsets, const int32_t* active_block,
                    int32_t T, int32_t B, int32_t E,
                    const reflex_alloc_params* p, int32_t* k_out,
                    int64_t* k_sum_out, int32_t* dev_status, void* stream);

/*
 * reflex_update_state — refinement-state update after one denoising forward
 * of block-wise inference (Sec. 3.1, Eq. 1): commits, confidence history and
 * active-block advance, in place, for the next forward's reflex_allocate.
 *
 * Per sequence s with a = active_block[s] (1 <= a <= num_blocks[s]) and J =
 * the masked positions of block a:
 *   - C = {i in J : conf_new[i] >= theta_commit} is committed (masked -> 0);
 *     if C is empty and J is not, the most confident member of J (lower
 *     position on ties) is committed instead;
 *   - every position masked during the forward shifts its history:
 *     conf_prev2 <- conf_prev1, conf_prev1 <- conf_new, hist_len <-
 *     min(hist_len + 1, 2);
 *   - when no position of block a is left masked, active_block[s] = a + 1.
 * A sequence with active_block[s] > num_blocks[s] is finished and untouched.
 *
 *   conf_new        [T] fp32  c^t of the forward (read where masked).
 *   conf_prev1/2    [T] fp32  in/out, as in reflex_allocate.
 *   hist_len        [T] u8    in/out.
 *   masked          [T] u8    in/out.
 *   block_id        [T] int32, seq_offsets [B+1]: as in reflex_allocate.
 *   active_block    [B] int32 in/out.
 *   num_blocks      [B] int32 Q of each sequence (its last target block).
 *   theta_commit    commitment threshold of Eq. 1 (Sec. 5.1: 0.9).
 *   committed_out   [B] int32 nullable: positions committed in each sequence.
 *   dev_status      [1] int32 nullable; error bits are OR-ed in (not cleared).
 * Device buffers, one CTA per sequence; returns REFLEX_EINVAL for null
 * pointers, T < 0, B < 1 or a non-finite theta_commit.
 */
int reflex_update_state(const float* conf_new, float* conf_prev1, float* conf_prev2,
                        uint8_t* hist_len, uint8_t* masked, const int32_t* block_id,
                        const int32_t* seq_offsets, int32_t* active_block,
                        const int32_t* num_blocks, int32_t T, int32_t B,
                        float theta_commit, int32_t* committed_out,
                        int32_t* dev_status, void* stream);

/* Device pointers into the workspace after a forward (the routing record). */
typedef struct {
    int32_t* ids;     /* [T, k_max] selected experts in router rank order,
                         -1 in slots j >= k_i                               */
    float* alpha;     /* [T, k_max] normalised router weights, 0 padded     */
    int32_t* counts;  /* [E] pairs per expert                               */
    int32_t* offsets; /* [E+1] first pair row of each expert                */
    int32_t* perm;    /* [sum k] pair rows: token * k_max + slot, ordered by
                         (expert, token)                                    */
    int32_t* row_of;  /* [T, k_max] pair row of (token, slot), -1 unused    */
    int32_t* totals;  /* [2] device: sum k (pairs), number of 128-row tiles */
    float* scores;    /* [T, E] router scores r_i (fp32), valid after the
                         ROUTE stage: the fma chain of reflex_moe_forward for
                         every expert that could be selected (all experts
                         with REFLEX_FLAG_EXACT_SCORES or fp32), tensor-core
                         estimates for the others                           */
} reflex_route_record;

/* Bytes of workspace reflex_moe_forward needs for these shapes (0 if the
 * shapes are invalid).  Sized for the worst case T * k_max pairs, so the
 * forward never reads back the realised sum of k.  Never decreases as T
 * grows (other shapes fixed): a workspace sized for T serves every smaller
 * batch. */
size_t reflex_moe_workspace_size(int32_t dtype, int32_t T, int32_t d,
                                 int32_t E, int32_t inter,
                                 int32_t shared_inter, int32_t k_max);

/*
 * reflex_moe_forward — the variable-count MoE layer, Eq. 2 (Sec. 3.2):
 *   out_i = sum_{e in TopK(r_i, k_i)} alpha_{i,e} E_e(h_i)  [+ shared(h_i)]
 * with r_i = h_i W_r^T (fp32; each score is the sequential fused
 * multiply-add chain over the hidden index from +0), TopK ties broken to the
 * lower expert index, and SwiGLU experts
 *   E_e(h) = (silu(h W_g,e^T) * (h W_u,e^T)) W_d,e^T.
 * The TopK is decided on the canonical chain's scores.  bf16 layers with
 * renormalised weights screen first: tensor-core scores z~ with an interval
 * z~ -/+ (gamma_d + 2^-12 + (s+1) 2^-24) ||h_i|| ||w_e|| (gamma_d = d u /
 * (1 - d u), u = 2^-24, s split-K slices) that holds both the chain's score
 * and the exact product; experts whose interval lies below the k_i-th
 * largest lower end cannot be selected, all others are recomputed with the
 * chain.  This assumes the tensor cores' fp32 accumulation errs by at most
 * 2^-12 sum_k |h_k w_k|; REFLEX_FLAG_EXACT_SCORES computes every score with
 * the chain instead.
 *
 *   dtype           REFLEX_DTYPE_F32 or REFLEX_DTYPE_BF16 (all float arrays).
 *   hidden          [T, d]
 *   w_router        [E, d]
 *   w_gate_up       [E, 2*inter, d]: rows [0, inter) gate, [inter, 2*inter) up
 *   w_down          [E, d, inter]
 *   shared_gate_up  [2*shared_inter, d], nullable (with shared_inter = 0)
 *   shared_down     [d, shared_inter]
 *   k               [T] int32 counts (from reflex_allocate or any rule);
 *                   each must lie in [1, min(k_max, E)] (else the device
 *                   error word gets REFLEX_EKRANGE and the count is clamped).
 *   flags           REFLEX_FLAG_* | REFLEX_STAGE_* (see above).
 *   workspace       >= reflex_moe_workspace_size(...) bytes, 256-B aligned.
 *   ws_bytes        the workspace's size in bytes; smaller than
 *                   reflex_moe_workspace_size(...) for this call's shapes:
 *                   REFLEX_EWORKSPACE, nothing enqueued.
 *   out             [T, d] output.
 *   rec             HOST struct, nullable: receives device pointers into the
 *                   workspace (no copy is made).
 * T == 0 launches no kernel; the workspace header (error word, totals) is
 * cleared in stream order, so reflex_moe_status reports this call.
 * Shape rules: T >= 0, d % 64 == 0, 1 <= E <= 1024, 1 <= k_max <= 32,
 * inter % 64 == 0, shared_inter % 64 == 0.  The bf16 tcgen05 path also needs
 * d % 256 == 0 and inter, shared_inter % 128 == 0 (else REFLEX_EUNSUPPORTED
 * unless REFLEX_FLAG_SIMT_EXPERTS is given).
 */
int reflex_moe_forward(int32_t dtype, const void* hidden, const void* w_router,
                       const void* w_gate_up, const void* w_down,
                       const void* shared_gate_up, const void* shared_down,
                       int32_t shared_inter, const int32_t* k, int32_t T,
                       int32_t d, int32_t E, int32_t inter, int32_t k_max,
                       uint32_t flags, void* workspace, size_t ws_bytes,
                       void* out, reflex_route_record* rec, void* stream);

/*
 * reflex_step — one denoising forward's hot path in one call: the per-token
 * counts of reflex_allocate (Eq. 5, Eq. 6-9, clip to [K_min, K_max]) for the
 * state arrays, then reflex_moe_forward with those counts (Eq. 2).  Every
 * output equals, bit for bit, that of reflex_allocate followed by
 * reflex_moe_forward on the same stream with the same arguments.  The
 * router scores do not depend on the counts, so the count kernel is launched
 * right behind the score kernel and runs beside it; the TopK selection waits
 * for both.
 *
 *   conf_prev1 .. active_block, B, p, k_out, k_sum_out: as for
 *                   reflex_allocate (T is the forward's T); alloc_status is
 *                   its device error word (nullable; stored or cleared by the
 *                   call, then OR-ed), separate from the forward's error word
 *                   in the workspace.
 *   dtype .. rec:   as for reflex_moe_forward; the counts read by the forward
 *                   are k_out (written by this call).
 * Ownership and errors: every pointer except rec and p is device memory owned
 * by the caller; nothing is allocated.  Any argument error of either half
 * returns its status before anything is launched.  The REFLEX_STAGE_* bits of
 * flags select the forward's stages as for reflex_moe_forward; the counts are
 * computed in every case.
 * With a score rule (p->count_rule TOP_P or EXPERT_THRESHOLD) the counts come
 * from the forward's own router scores: the TopK selection derives each k_i
 * from z_i (as reflex_allocate with those scores would), writes it to k_out
 * and selects with it; the state arrays are not read (they may be NULL), and
 * the ROUTE stage must be among the selected stages (else REFLEX_EINVAL).
 */
int reflex_step(const float* conf_prev1, const float* conf_prev2, const uint8_t* hist_len,
                const uint8_t* masked, const int32_t* block_id, const int32_t* seq_offsets,
                const int32_t* active_block, int32_t B, const reflex_alloc_params* p,
                int32_t* k_out, int64_t* k_sum_out, int32_t* alloc_status,
                int32_t dtype, const void* hidden, const void* w_router,
                const void* w_gate_up, const void* w_down, const void* shared_gate_up,
                const void* shared_down, int32_t shared_inter, int32_t T, int32_t d,
                int32_t E, int32_t inter, int32_t k_max, uint32_t flags, void* workspace,
                size_t ws_bytes, void* out, reflex_route_record* rec, void* stream);

/*
 * reflex_route_noalloc — the routing step of reflex_moe_forward (router
 * scores, TopK(r_i, k_i), router weights) for callers that cannot allocate
 * device memory: code inside a framework that owns the device allocator and
 * forbids side allocations, plugins limited to the buffers they are handed,
 * or processes where cudaMalloc is not allowed after start-up.  The paper has
 * no counterpart; it is a deployment convenience.
 *
 * The one scratch buffer of this step, the fp32 score matrix [T, E], lives
 * in a fixed array inside the library's device memory
 * (REFLEX_NOALLOC_MAX_SCORES floats = 4 MiB, held on every GPU that uses the
 * library until the process exits).  Nothing is allocated or freed.
 *   ids_out    [T, k_max] int32, alpha_out [T, k_max] fp32: same meaning and
 *              values as the ids / alpha of reflex_route_record.
 *   dev_status nullable device error word: cleared with a 4-byte memset in
 *              stream order before this call's kernels (also when T == 0),
 *              then OR-ed with error bits; read it with reflex_read_status.
 * Returns REFLEX_EWORKSPACE when T * E > REFLEX_NOALLOC_MAX_SCORES, and
 * REFLEX_EINVAL for the shape errors of reflex_moe_forward.  The first call
 * on each device looks up the array's address; make it before any stream
 * capture.  All calls share the array: calls whose GPU work overlaps in time
 * race on it and must be serialised.
 */
#define REFLEX_NOALLOC_MAX_SCORES (1 << 20)
int reflex_route_noalloc(int32_t dtype, const void* hidden,
                         const void* w_router, const int32_t* k, int32_t T,
                         int32_t d, int32_t E, int32_t k_max, uint32_t flags,
                         int32_t* ids_out, float* alpha_out,
                         int32_t* dev_status, void* stream);

/* Synchronises `stream` and returns the status recorded in the workspace's
 * device error word by the last forward (REFLEX_OK if clean). */
int reflex_moe_status(const void* workspace, void* stream);

/* Same for a caller-owned device error word (e.g. reflex_allocate's). */
int reflex_read_status(const int32_t* dev_status, void* stream);

/* Bounded-wait self-test: launches one block that waits on an mbarrier no
 * one arrives at, with a limit of `limit_us` microseconds (1..100000), then
 * records REFLEX_ETIMEOUT in dev_status and returns.  Exercises the same
 * wait routine the tcgen05 pipeline uses; nothing hangs. */
int reflex_selftest_wait_timeout(int32_t* dev_status, uint32_t limit_us,
                                 void* stream);

/* Human-readable status. */
const char* reflex_status_string(int status);

/* Version of this ABI (major * 100 + minor). */
int reflex_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* REFLEX_H */
