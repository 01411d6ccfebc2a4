/*
 * reflex_oracle.c — plain, slow CPU oracle for the REFLEX per-forward MoE path.
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / reference legs of bench.py may load this library.  The
 * product path (include/reflex.h, paper_2608_01784_gb300/) never calls it and
 * shares no code, header, table or constant with it.
 *
 * What it computes (paper section / equation it follows):
 *   oracle_exp_f32       own fp32 exp: Cody-Waite argument reduction (Cody &
 *                        Waite 1980) + degree-7 Taylor polynomial, separate
 *                        IEEE operations only.  Used by the FPS sigmoids.
 *   oracle_allocate      Refinement-Role Budgeting (Sec. 4.2, Eq. 5) then
 *                        Frontier-Guided Expert Reallocation (Sec. 4.3,
 *                        forecast, Eq. 6-8 and Eq. 9), then the clip of every
 *                        count to [K_min, K_max] required by Eq. 3.
 *   oracle_update_state  block-wise inference after one forward (Sec. 3.1,
 *                        Eq. 1): threshold commits in the active block (the
 *                        most confident one when none reaches the threshold),
 *                        the confidence history of every masked position, and
 *                        the active-block advance once the block is resolved.
 *   oracle_allocate_ex   the same with the ablations of App. C: the rank key
 *                        of the Eq. 9 groups (FPS, F only, P only, c^{t-1},
 *                        1 - c^{t-1}) and Role-Shuffled RRB (a seeded
 *                        permutation of each sequence's counts; its keys come
 *                        from splitmix64, Steele, Lea and Flood 2014).
 *   oracle_router_logits router scores r = h . W_r (Sec. 3.2) as a sequential
 *                        fp32 fused-multiply-add chain over the hidden index,
 *                        k = 0 .. d-1, starting from +0 (the summation-order
 *                        contract the GPU router also follows).
 *   oracle_select        TopK_e(r, k_i) of Eq. 2 (ties: lower expert index)
 *                        and the normalised router weight alpha in fp64.
 *   oracle_rule_counts   the counts of the threshold-based comparison
 *                        methods (App. B): Top-p (smallest router-ranked
 *                        prefix whose routing mass reaches p) and Expert-
 *                        Threshold routing (experts whose routing mass
 *                        exceeds a threshold), clipped to the count bounds.
 *   oracle_permutation   token-expert pairs sorted by (expert, token): the
 *                        per-expert row ranges that execute Eq. 2 sparsely.
 *   oracle_moe_tokens    Eq. 2 for a list of tokens: sum over selected experts
 *                        of alpha * SwiGLU expert, plus an optional always-on
 *                        shared expert (alpha = 1), in fp64.
 *
 * Floating-point contract: build with -O2 -ffp-contract=off so that every
 * a*b+c written below is two rounded operations unless fmaf() is called.
 *
 * Parity pins live in tests/test_oracle_pins.py; every function above has at
 * least one pin that does not re-run the function's own formula.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OR_OK 0
#define OR_EINVAL 1

/* ------------------------------------------------------------------------ */
/* bf16 helpers: a bf16 value is the top 16 bits of an IEEE binary32.        */
/* ------------------------------------------------------------------------ */
static float or_bf16_to_f32(uint16_t b) {
    uint32_t u = ((uint32_t)b) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return f;
}

static float or_load(const void* base, int32_t dtype, int64_t idx) {
    /* dtype 0 = fp32 element, 1 = bf16 element (widened exactly) */
    if (dtype == 0) return ((const float*)base)[idx];
    return or_bf16_to_f32(((const uint16_t*)base)[idx]);
}

/* ------------------------------------------------------------------------ */
/* exp in fp32 from a published method.                                      */
/*   x = k*ln2 + r,  k = round-half-even(x / ln2),  |r| <= ln2/2             */
/*   r computed with ln2 split in a high part of few bits (k*hi exact) and   */
/*   a low part (Cody & Waite 1980).                                         */
/*   e^r by its Taylor series to degree 7 in Horner form (truncation error   */
/*   below 2^-27 relative on |r| <= ln2/2).                                  */
/*   Result scaled by 2^k as two exact power-of-two factors so that neither  */
/*   factor overflows and a subnormal result is rounded once.                */
/* ------------------------------------------------------------------------ */
static float or_pow2i(int32_t e) {
    /* 2^e for e in [-126, 127], built from its bit pattern */
    uint32_t u = ((uint32_t)(e + 127)) << 23;
    float f;
    memcpy(&f, &u, sizeof f);
    return f;
}

float oracle_exp_f32(float x) {
    const float inv_ln2 = 1.44269502162933349609375f;      /* fp32(1/ln 2) */
    const float ln2_hi = 0.693145751953125f;               /* 0x3F317200   */
    const float ln2_lo = 1.428606765330187045037746429443359375e-06f;
    if (x != x) return x;
    if (x >= 89.0f) return INFINITY;
    if (x <= -104.0f) return 0.0f;
    float t = x * inv_ln2;
    float kf = rintf(t); /* default rounding mode: nearest, ties to even */
    int32_t k = (int32_t)kf;
    float r = x - kf * ln2_hi;
    r = r - kf * ln2_lo;
    /* Taylor coefficients 1/n!, n = 7 .. 0 */
    float p = 1.98412701138295233249664306640625e-04f;    /* 1/5040 */
    p = p * r + 1.388888922519981861114501953125e-03f;      /* 1/720  */
    p = p * r + 8.33333376795053482055664062500000e-03f;   /* 1/120  */
    p = p * r + 4.16666679084300994873046875000000e-02f;   /* 1/24   */
    p = p * r + 1.66666671633720397949218750000000e-01f;   /* 1/6    */
    p = p * r + 0.5f;
    p = p * r + 1.0f;
    p = p * r + 1.0f;
    int32_t k1 = k >> 1; /* floor(k/2) for negative k as well */
    int32_t k2 = k - k1;
    float y = p * or_pow2i(k1);
    y = y * or_pow2i(k2);
    return y;
}

static float or_sigmoid(float x) {
    float e = oracle_exp_f32(-x);
    float den = 1.0f + e;
    return 1.0f / den;
}

/* ------------------------------------------------------------------------ */
/* Frontier-Progress Score of one token (Sec. 4.3).                          */
/* hist: number of past confidence observations available (0, 1, 2+).       */
/* Operation order (all fp32, one rounding per operation):                  */
/*   v    = hist>=2 ? c1 - c2 : 0                    lagged change          */
/*   vbar = clip(v, -w/2, w/2)                                              */
/*   chat = clip(c1 + vbar, 0, 1)                    forecast               */
/*   F    = sig(((chat - theta) + w) / tau) * sig((theta - chat) / tau) Eq.6 */
/*   P    = hist>=2 ? sig((v_ref - vbar) / tau) : 1                   Eq.7 */
/*   S    = F * P                                                     Eq.8 */
/* ------------------------------------------------------------------------ */
static void or_frontier_progress(float c1, float c2, int32_t hist, float theta,
                                 float w_cf, float v_ref, float tau,
                                 float* F_out, float* P_out) {
    float v = (hist >= 2) ? (c1 - c2) : 0.0f;
    float half_w = w_cf * 0.5f;
    float vbar = fminf(fmaxf(v, -half_w), half_w);
    float chat = fminf(fmaxf(c1 + vbar, 0.0f), 1.0f);
    float x1 = ((chat - theta) + w_cf) / tau;
    float x2 = (theta - chat) / tau;
    *F_out = or_sigmoid(x1) * or_sigmoid(x2);
    *P_out = (hist >= 2) ? or_sigmoid((v_ref - vbar) / tau) : 1.0f;
}

float oracle_fps(float c1, float c2, int32_t hist, float theta, float w_cf,
                 float v_ref, float tau) {
    float F, P;
    or_frontier_progress(c1, c2, hist, theta, w_cf, v_ref, tau, &F, &P);
    return F * P;
}

/* Rank key of a J_h member under each signal of the App. C ablation:      */
/*   0 FPS: F * P     1 Frontier: F     2 Progress: P                      */
/*   3 Confidence: c^{t-1}     4 Uncertainty: 1 - c^{t-1} (fp32)           */
float oracle_rank_key(int32_t signal, float c1, float c2, int32_t hist,
                      float theta, float w_cf, float v_ref, float tau) {
    float F, P;
    if (signal == 3) return c1;
    if (signal == 4) return 1.0f - c1;
    or_frontier_progress(c1, c2, hist, theta, w_cf, v_ref, tau, &F, &P);
    if (signal == 1) return F;
    if (signal == 2) return P;
    return F * P;
}

/* splitmix64 output number n (n >= 1) of the stream seeded with seed: the  */
/* state is seed + n * golden gamma, the output its "mix13" finaliser.      */
uint64_t oracle_splitmix64(uint64_t seed, uint64_t n) {
    uint64_t z = seed + n * 0x9e3779b97f4a7c15ULL;
    z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ULL;
    z = (z ^ (z >> 27)) * 0x94d049bb133111ebULL;
    return z ^ (z >> 31);
}

/* ------------------------------------------------------------------------ */
/* Allocation: RRB (Eq. 5) then FGER (Eq. 9) then clip to [K_min, K_max].   */
/* Per sequence s (tokens seq_off[s] .. seq_off[s+1]-1, active block a):     */
/*  1. k_i = H(|b(i) - a|), prompt tokens carry b = 0.                       */
/*  2. J_h = masked tokens of block a with at least one past confidence.     */
/*     Other tokens of block a keep K_cur = H(0).                            */
/*  3. Rank J_h by (S descending, position ascending); n = floor(q |J_h|);   */
/*     the first n get K_cur + delta_cur, the last n get K_cur - delta_cur.  */
/*  4. Clip every k to [K_min, K_max].                                       */
/* Returns OR_EINVAL when an active block index is < 1.                      */
/* s_out (nullable) receives S for members of J_h and NaN elsewhere.         */
/* ------------------------------------------------------------------------ */
static int32_t or_role_count(int32_t dist, int32_t k_base, int32_t d_role) {
    if (dist <= 1) return k_base + d_role;
    if (dist == 2) return k_base;
    return k_base - d_role;
}

typedef struct {
    uint32_t key;
    int32_t pos;
} or_key_pos;

static int or_cmp_key_pos(const void* a, const void* b) {
    const or_key_pos* x = (const or_key_pos*)a;
    const or_key_pos* y = (const or_key_pos*)b;
    if (x->key != y->key) return x->key < y->key ? -1 : 1;
    return x->pos < y->pos ? -1 : (x->pos > y->pos ? 1 : 0);
}

int oracle_allocate_ex(const float* conf1, const float* conf2,
                       const uint8_t* hist_len, const uint8_t* masked,
                       const int32_t* block_id, const int32_t* seq_off,
                       const int32_t* active_block, int32_t T, int32_t B,
                       int32_t k_min, int32_t k_base, int32_t k_max,
                       int32_t delta_role, int32_t delta_cur, float q,
                       float theta, float w_cf, float v_ref, float tau,
                       int32_t signal, int32_t role_shuffle, uint64_t shuffle_seed,
                       int32_t* k_out, float* s_out) {
    if (T < 0 || B < 0) return OR_EINVAL;
    if (T > 0 && seq_off[B] != T) return OR_EINVAL;
    for (int32_t i = 0; i < T; ++i) {
        if (s_out) s_out[i] = NAN;
    }
    for (int32_t s = 0; s < B; ++s) {
        int32_t lo = seq_off[s], hi = seq_off[s + 1];
        int32_t a = active_block[s];
        if (a < 1) return OR_EINVAL;
        int32_t k_cur = k_base + delta_role;
        /* step 1: role map */
        for (int32_t i = lo; i < hi; ++i) {
            int32_t dist = abs(block_id[i] - a);
            k_out[i] = or_role_count(dist, k_base, delta_role);
        }
        /* step 2: collect J_h with its score */
        int32_t nj = 0;
        int32_t* idx = (int32_t*)malloc(sizeof(int32_t) * (size_t)(hi - lo + 1));
        float* sc = (float*)malloc(sizeof(float) * (size_t)(hi - lo + 1));
        for (int32_t i = lo; i < hi; ++i) {
            if (block_id[i] == a && masked[i] && hist_len[i] >= 1) {
                idx[nj] = i;
                sc[nj] = oracle_rank_key(signal, conf1[i], conf2[i], hist_len[i],
                                         theta, w_cf, v_ref, tau);
                if (s_out) s_out[i] = sc[nj];
                ++nj;
            }
        }
        /* step 3: sort J_h by (S desc, position asc) with insertion sort */
        for (int32_t x = 1; x < nj; ++x) {
            int32_t ci = idx[x];
            float cs = sc[x];
            int32_t y = x - 1;
            while (y >= 0 && (sc[y] < cs || (sc[y] == cs && idx[y] > ci))) {
                idx[y + 1] = idx[y];
                sc[y + 1] = sc[y];
                --y;
            }
            idx[y + 1] = ci;
            sc[y + 1] = cs;
        }
        int32_t n = (int32_t)floorf(q * (float)nj);
        for (int32_t r = 0; r < nj; ++r) {
            int32_t i = idx[r];
            int32_t k = k_cur;
            if (r < n) k = k_cur + delta_cur;
            else if (r >= nj - n) k = k_cur - delta_cur;
            k_out[i] = k;
        }
        free(idx);
        free(sc);
        /* step 4: clip */
        for (int32_t i = lo; i < hi; ++i) {
            int32_t k = k_out[i];
            if (k < k_min) k = k_min;
            if (k > k_max) k = k_max;
            k_out[i] = k;
        }
        /* step 5 (Role-Shuffled RRB): sort the positions by (key, position);
           the token in sorted place r receives the count of position lo + r */
        if (role_shuffle && hi > lo) {
            int32_t len = hi - lo;
            or_key_pos* kp = (or_key_pos*)malloc(sizeof(or_key_pos) * (size_t)len);
            int32_t* old = (int32_t*)malloc(sizeof(int32_t) * (size_t)len);
            for (int32_t r = 0; r < len; ++r) {
                kp[r].key = (uint32_t)(oracle_splitmix64(shuffle_seed,
                                                         (uint64_t)(lo + r) + 1) >> 32);
                kp[r].pos = lo + r;
                old[r] = k_out[lo + r];
            }
            qsort(kp, (size_t)len, sizeof(or_key_pos), or_cmp_key_pos);
            for (int32_t r = 0; r < len; ++r) k_out[kp[r].pos] = old[r];
            free(kp);
            free(old);
        }
    }
    return OR_OK;
}

int oracle_allocate(const float* conf1, const float* conf2,
                    const uint8_t* hist_len, const uint8_t* masked,
                    const int32_t* block_id, const int32_t* seq_off,
                    const int32_t* active_block, int32_t T, int32_t B,
                    int32_t k_min, int32_t k_base, int32_t k_max,
                    int32_t delta_role, int32_t delta_cur, float q,
                    float theta, float w_cf, float v_ref, float tau,
                    int32_t* k_out, float* s_out) {
    return oracle_allocate_ex(conf1, conf2, hist_len, masked, block_id, seq_off,
                              active_block, T, B, k_min, k_base, k_max, delta_role,
                              delta_cur, q, theta, w_cf, v_ref, tau, 0, 0, 0,
                              k_out, s_out);
}

/* ------------------------------------------------------------------------ */
/* Router scores: z[t,e] = sum_k h[t,k] * W_r[e,k], as the chain             */
/*   acc = +0;  for k = 0..d-1: acc = fmaf(h[t,k], W_r[e,k], acc)            */
/* Inputs are widened exactly from bf16 when dtype = 1.                      */
/* ------------------------------------------------------------------------ */
/* ------------------------------------------------------------------------ */
/* Refinement-state update after forward t (Sec. 3.1, Eq. 1), per sequence: */
/*  J = masked positions of the active block a (skip when a > Q).           */
/*  C = {i in J : c_i >= theta}; if C is empty and J is not, C = {the i in J */
/*  with the largest c_i, lowest position among equals}.  x_i <- candidate  */
/*  for i in C (masked_i = 0); J \ C stays masked; other positions keep.   */
/*  History: every position masked during the forward got the prediction   */
/*  c_i: c^{t-2} <- c^{t-1}, c^{t-1} <- c_i, hist <- min(hist + 1, 2).      */
/*  If block a has no masked position left, a <- a + 1.                     */
/* committed (nullable) receives |C| per sequence.                           */
/* ------------------------------------------------------------------------ */
int oracle_update_state(const float* conf_new, float* conf1, float* conf2,
                        uint8_t* hist_len, uint8_t* masked, const int32_t* block_id,
                        const int32_t* seq_off, int32_t* active, const int32_t* num_blocks,
                        int32_t T, int32_t B, float theta, int32_t* committed) {
    if (T < 0 || B < 0) return OR_EINVAL;
    if (T > 0 && seq_off[B] != T) return OR_EINVAL;
    for (int32_t s = 0; s < B; ++s) {
        int32_t lo = seq_off[s], hi = seq_off[s + 1];
        int32_t a = active[s];
        if (committed) committed[s] = 0;
        if (a < 1) return OR_EINVAL;
        if (a > num_blocks[s]) continue;                  /* finished */
        /* the masked set seen by the forward, before any commit */
        uint8_t* was_masked = (uint8_t*)malloc((size_t)(hi - lo + 1));
        for (int32_t i = lo; i < hi; ++i) was_masked[i - lo] = masked[i];
        int32_t nj = 0, nc = 0, best = -1;
        for (int32_t i = lo; i < hi; ++i) {
            if (!was_masked[i - lo] || block_id[i] != a) continue;
            ++nj;
            if (best < 0 || conf_new[i] > conf_new[best]) best = i;  /* first max */
            if (conf_new[i] >= theta) {
                masked[i] = 0;
                ++nc;
            }
        }
        if (nj > 0 && nc == 0) {
            masked[best] = 0;
            nc = 1;
        }
        for (int32_t i = lo; i < hi; ++i) {
            if (!was_masked[i - lo]) continue;
            conf2[i] = conf1[i];
            conf1[i] = conf_new[i];
            hist_len[i] = (uint8_t)(hist_len[i] >= 2 ? 2 : hist_len[i] + 1);
        }
        if (nj - nc == 0) active[s] = a + 1;
        if (committed) committed[s] = nc;
        free(was_masked);
    }
    return OR_OK;
}

void oracle_router_logits(int32_t dtype, const void* hidden,
                          const void* w_router, int32_t T, int32_t d,
                          int32_t E, float* z) {
#pragma omp parallel for schedule(static)
    for (int32_t t = 0; t < T; ++t) {
        for (int32_t e = 0; e < E; ++e) {
            float acc = 0.0f;
            for (int32_t k = 0; k < d; ++k) {
                float h = or_load(hidden, dtype, (int64_t)t * d + k);
                float w = or_load(w_router, dtype, (int64_t)e * d + k);
                acc = fmaf(h, w, acc);
            }
            z[(int64_t)t * E + e] = acc;
        }
    }
}

/* ------------------------------------------------------------------------ */
/* TopK_e(z, k_t) with ties to the lower expert index, then alpha (fp64):    */
/*   p_e = exp(z_e - max z) / sum_e' exp(z_e' - max z)   (softmax over E)    */
/*   renorm = 1: alpha_j = p_{ids_j} / sum over the selected set             */
/*   renorm = 0: alpha_j = p_{ids_j}                                         */
/* ids/alpha are [T, k_max]; slots j >= k_t hold -1 / 0.                     */
/* Returns OR_EINVAL when some k_t is outside [1, min(k_max, E)].            */
/* ------------------------------------------------------------------------ */
int oracle_select(const float* z, const int32_t* k, int32_t T, int32_t E,
                  int32_t k_max, int32_t renorm, int32_t* ids,
                  double* alpha) {
    int32_t* order = (int32_t*)malloc(sizeof(int32_t) * (size_t)E);
    for (int32_t t = 0; t < T; ++t) {
        const float* zt = z + (int64_t)t * E;
        int32_t kt = k[t];
        if (kt < 1 || kt > k_max || kt > E) {
            free(order);
            return OR_EINVAL;
        }
        /* selection: repeatedly take the best remaining expert */
        for (int32_t e = 0; e < E; ++e) order[e] = e;
        for (int32_t j = 0; j < kt; ++j) {
            int32_t best = j;
            for (int32_t c = j + 1; c < E; ++c) {
                int32_t ec = order[c], eb = order[best];
                if (zt[ec] > zt[eb] || (zt[ec] == zt[eb] && ec < eb)) best = c;
            }
            int32_t tmp = order[j];
            order[j] = order[best];
            order[best] = tmp;
        }
        double zmax = (double)zt[order[0]];
        double all = 0.0, sel = 0.0;
        for (int32_t e = 0; e < E; ++e) all += exp((double)zt[e] - zmax);
        for (int32_t j = 0; j < kt; ++j) sel += exp((double)zt[order[j]] - zmax);
        for (int32_t j = 0; j < k_max; ++j) {
            int64_t o = (int64_t)t * k_max + j;
            if (j < kt) {
                double pe = exp((double)zt[order[j]] - zmax);
                ids[o] = order[j];
                alpha[o] = renorm ? pe / sel : pe / all;
            } else {
                ids[o] = -1;
                alpha[o] = 0.0;
            }
        }
    }
    free(order);
    return OR_OK;
}

/* ------------------------------------------------------------------------ */
/* Score-based count rules of the threshold-based comparison methods        */
/* (App. B): the count of token t comes from its router scores z_t alone.   */
/* The routing mass is the softmax of z_t over the E experts; the decision  */
/* is taken in fp32 in this order (the order the GPU follows):             */
/*   m   = max_e z_e                                                        */
/*   u_e = exp_f32(z_e - m)                          (oracle_exp_f32)      */
/*   S   : 32 lane sums s_l = ((0 + u_l) + u_{l+32}) + ..., l = 0 .. 31,    */
/*         then for o = 16, 8, 4, 2, 1 every s_l <- s_l + s_{l xor o};      */
/*         S = s_0                                                          */
/*   rule 1, Top-p: ranks j = 1, 2, ... by (z desc, e asc);                 */
/*         c_j = c_{j-1} + u_(j), c_0 = 0; k = the smallest j with          */
/*         c_j / S >= thr (E when no j reaches it)                         */
/*   rule 2, Expert threshold: k = #{e : u_e / S > thr}                    */
/* then k is clipped to [k_min, min(k_max, E)] (the paper: [1, 12]).       */
/* Returns OR_EINVAL for an unknown rule or bounds.                        */
/* ------------------------------------------------------------------------ */
int oracle_rule_counts(const float* z, int32_t T, int32_t E, int32_t rule,
                       float thr, int32_t k_min, int32_t k_max, int32_t* k_out) {
    if (E < 1 || (rule != 1 && rule != 2) || k_min < 1 || k_max < k_min) return OR_EINVAL;
    int32_t kcap = k_max < E ? k_max : E;
    int32_t klo = k_min < kcap ? k_min : kcap;
    float* u = (float*)malloc(sizeof(float) * (size_t)E);
    int32_t* order = (int32_t*)malloc(sizeof(int32_t) * (size_t)E);
    for (int32_t t = 0; t < T; ++t) {
        const float* zt = z + (int64_t)t * E;
        float m = zt[0];
        for (int32_t e = 1; e < E; ++e)
            if (zt[e] > m) m = zt[e];
        for (int32_t e = 0; e < E; ++e) u[e] = oracle_exp_f32(zt[e] - m);
        float lane[32];
        for (int32_t l = 0; l < 32; ++l) {
            float acc = 0.0f;
            for (int32_t e = l; e < E; e += 32) acc = acc + u[e];
            lane[l] = acc;
        }
        for (int32_t o = 16; o > 0; o >>= 1) {
            float nxt[32];
            for (int32_t l = 0; l < 32; ++l) nxt[l] = lane[l] + lane[l ^ o];
            for (int32_t l = 0; l < 32; ++l) lane[l] = nxt[l];
        }
        float S = lane[0];
        int32_t k;
        if (rule == 2) {
            k = 0;
            for (int32_t e = 0; e < E; ++e)
                if (u[e] / S > thr) ++k;
        } else {
            /* rank order: repeatedly the best remaining expert */
            for (int32_t e = 0; e < E; ++e) order[e] = e;
            k = E;
            float c = 0.0f;
            for (int32_t j = 0; j < E; ++j) {
                int32_t best = j;
                for (int32_t q = j + 1; q < E; ++q) {
                    int32_t eq = order[q], eb = order[best];
                    if (zt[eq] > zt[eb] || (zt[eq] == zt[eb] && eq < eb)) best = q;
                }
                int32_t tmp = order[j];
                order[j] = order[best];
                order[best] = tmp;
                c = c + u[order[j]];
                if (c / S >= thr) {
                    k = j + 1;
                    break;
                }
            }
        }
        if (k < klo) k = klo;
        if (k > kcap) k = kcap;
        k_out[t] = k;
    }
    free(u);
    free(order);
    return OR_OK;
}

/* ------------------------------------------------------------------------ */
/* Pair permutation: the pairs (t, j), j < k_t, ordered by expert, then by   */
/* token.  perm[p] = t * k_max + j; offsets[e] = first row of expert e;      */
/* row_of[t*k_max + j] = p (or -1 for unused slots).  Returns sum k_t.        */
/* ------------------------------------------------------------------------ */
int64_t oracle_permutation(const int32_t* ids, const int32_t* k, int32_t T,
                           int32_t E, int32_t k_max, int32_t* offsets,
                           int32_t* perm, int32_t* row_of) {
    int64_t pos = 0;
    for (int64_t o = 0; o < (int64_t)T * k_max; ++o) row_of[o] = -1;
    for (int32_t e = 0; e < E; ++e) {
        offsets[e] = (int32_t)pos;
        for (int32_t t = 0; t < T; ++t) {
            for (int32_t j = 0; j < k[t]; ++j) {
                int64_t o = (int64_t)t * k_max + j;
                if (ids[o] == e) {
                    perm[pos] = (int32_t)o;
                    row_of[o] = (int32_t)pos;
                    ++pos;
                }
            }
        }
    }
    offsets[E] = (int32_t)pos;
    return pos;
}

/* ------------------------------------------------------------------------ */
/* One SwiGLU expert on one token, fp64 accumulation:                        */
/*   g_c = h . Wg[c], u_c = h . Wu[c], a_c = silu(g_c) * u_c,                */
/*   y_n = sum_c a_c * Wd[n, c]                                              */
/* w_gate_up rows [0, inter) are gate, [inter, 2 inter) are up; w_down is    */
/* [d, inter].  y (length d) is accumulated with weight scale.               */
/* ------------------------------------------------------------------------ */
static void or_expert_accumulate(int32_t dtype, const double* h,
                                 const void* w_gate_up, const void* w_down,
                                 int64_t gu_base, int64_t dn_base, int32_t d,
                                 int32_t inter, double scale, double* act,
                                 double* y) {
    for (int32_t c = 0; c < inter; ++c) {
        double g = 0.0, u = 0.0;
        for (int32_t kk = 0; kk < d; ++kk) {
            g += h[kk] * (double)or_load(w_gate_up, dtype, gu_base + (int64_t)c * d + kk);
            u += h[kk] * (double)or_load(w_gate_up, dtype, gu_base + (int64_t)(inter + c) * d + kk);
        }
        double silu = g / (1.0 + exp(-g));
        act[c] = silu * u;
    }
    for (int32_t n = 0; n < d; ++n) {
        double acc = 0.0;
        for (int32_t c = 0; c < inter; ++c)
            acc += act[c] * (double)or_load(w_down, dtype, dn_base + (int64_t)n * inter + c);
        y[n] += scale * acc;
    }
}

/* ------------------------------------------------------------------------ */
/* Eq. 2 for the listed tokens:                                              */
/*   out[r, :] = sum_{j < k_t} alpha[t, j] * E_{ids[t, j]}(h_t)              */
/*             + shared(h_t)            (when shared_inter > 0)              */
/* with t = tokens[r].  out is [n_tokens, d] fp64.                           */
/* ------------------------------------------------------------------------ */
void oracle_moe_tokens(int32_t dtype, const void* hidden, const void* w_gate_up,
                       const void* w_down, const void* shared_gate_up,
                       const void* shared_down, int32_t shared_inter,
                       const int32_t* ids, const double* alpha,
                       const int32_t* k, const int32_t* tokens,
                       int32_t n_tokens, int32_t d, int32_t inter,
                       int32_t k_max, double* out) {
#pragma omp parallel for schedule(dynamic, 1)
    for (int32_t r = 0; r < n_tokens; ++r) {
        int32_t t = tokens[r];
        double* h = (double*)malloc(sizeof(double) * (size_t)d);
        int32_t amax = inter > shared_inter ? inter : shared_inter;
        double* act = (double*)malloc(sizeof(double) * (size_t)(amax > 0 ? amax : 1));
        double* y = out + (int64_t)r * d;
        for (int32_t kk = 0; kk < d; ++kk) {
            h[kk] = (double)or_load(hidden, dtype, (int64_t)t * d + kk);
            y[kk] = 0.0;
        }
        for (int32_t j = 0; j < k[t]; ++j) {
            int64_t o = (int64_t)t * k_max + j;
            int64_t e = ids[o];
            or_expert_accumulate(dtype, h, w_gate_up, w_down,
                                 e * 2 * (int64_t)inter * d,
                                 e * (int64_t)d * inter, d, inter, alpha[o],
                                 act, y);
        }
        if (shared_inter > 0)
            or_expert_accumulate(dtype, h, shared_gate_up, shared_down, 0, 0,
                                 d, shared_inter, 1.0, act, y);
        free(h);
        free(act);
    }
}

int oracle_num_threads(void) {
#ifdef _OPENMP
    extern int omp_get_max_threads(void);
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* Threads used by the OpenMP loops from now on (timing the oracle on one  */
/* core and on all cores); no effect without OpenMP.                       */
void oracle_set_num_threads(int n) {
#ifdef _OPENMP
    extern void omp_set_num_threads(int);
    if (n >= 1) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

/* Array forms used by the pins and by the parity tests. */
void oracle_exp_f32_n(const float* x, float* y, int64_t n) {
    for (int64_t i = 0; i < n; ++i) y[i] = oracle_exp_f32(x[i]);
}

void oracle_fps_n(const float* c1, const float* c2, const uint8_t* hist,
                  int64_t n, float theta, float w_cf, float v_ref, float tau,
                  float* s) {
    for (int64_t i = 0; i < n; ++i)
        s[i] = oracle_fps(c1[i], c2[i], hist[i], theta, w_cf, v_ref, tau);
}

/* ------------------------------------------------------------------------ */
/* Rounding to bf16 (8 significant bits, fp32 exponent range), nearest with  */
/* ties to even, from fp64: x = m 2^e with m in [0.5, 1); the significand    */
/* m 2^8 is rounded to an integer in the current (nearest-even) mode.        */
/* ------------------------------------------------------------------------ */
static uint16_t or_bf16_from_f64(double x) {
    if (x != x) return 0x7FC0;
    if (x == 0.0) return signbit(x) ? 0x8000 : 0x0000;
    int e;
    double m = frexp(x, &e);            /* |m| in [0.5, 1) */
    double q = rint(ldexp(m, 8));       /* 8 significant bits */
    double r = ldexp(q, e - 8);         /* exactly a bf16 value (normal range) */
    float f = (float)r;                 /* exact */
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    return (uint16_t)(u >> 16);
}

void oracle_bf16_from_f64_n(const double* x, int64_t n, uint16_t* out) {
    for (int64_t i = 0; i < n; ++i) out[i] = or_bf16_from_f64(x[i]);
}

/* Residual update of a stacked layer: next = bf16(h + out) (h bf16 bits,   */
/* out the fp64 layer output).                                             */
void oracle_residual_bf16(const uint16_t* h, const double* out, int64_t n,
                          uint16_t* next) {
    for (int64_t i = 0; i < n; ++i)
        next[i] = or_bf16_from_f64((double)or_bf16_to_f32(h[i]) + out[i]);
}
