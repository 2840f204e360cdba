/*
 * eti_oracle.c -- plain, slow, fp64 CPU oracle of the entropic-time decode step.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may call, link or
 * load this file: only the test suite, the smoke check and the benchmark's
 * CPU-baseline / reference leg use it.  It shares no code, header, table or
 * helper with the CUDA kernels; it is written from the definitions of
 * "Entropic-Time Inference" (arXiv 2603.03310) and the published
 * description of the Philox4x32-10 generator (Salmon et al., SC'11).
 *
 * Everything is computed in double precision with direct two-pass loops
 * (no online softmax, no fusion).  bf16 inputs arrive as their 16-bit
 * patterns and are widened exactly (bits << 16 -> float -> double).
 * Loops over independent sequences / heads carry an OpenMP pragma so the
 * oracle finishes in seconds at full sizes; the arithmetic inside each
 * iteration is untouched by it.
 *
 * Readings of the paper that the code below fixes (each also stated where
 * it is used):
 *   R1  temperature law sign: T' = clip(T * exp(sigma*eta*(H - H*)));
 *       sigma = -1 restores (H grows with T), sigma = +1 is the printed form.
 *   R2  entropy, sample and surprisal all use the incoming T_t; T' is for t+1.
 *   R4  block surprisal I(v_i) := -log a_i (attention as a distribution over
 *       the values), so sum_b I_b is the attention entropy (score mode A, the
 *       default).  The other readings of "the surprisal associated with the
 *       value vector": mode E, I(v_i) := the stored surprisal -log p(x_i |
 *       x_<i) of the token at position i (recorded when it was generated);
 *       mode M, I(v_i) := 1, so I_b is the block's attention mass.
 *   R5  one keep decision per (sequence, kv head, block); group score is the
 *       max over the query heads that share the kv head.
 *   R6  threshold applies to the normalised score n_b * I_b / sum_b' I_b'.
 *   R7  keep iff score >= theta, or the block is among the first
 *       min(B_min, n_b) blocks ordered by (score desc, block index asc).
 *   R8  attention restricted to the kept blocks renormalises over them.
 *   R13 the Section 5 guards: calibration rescales the logits by 1 / T_cal
 *       before the step (entropy and draw use z / (T_cal T_t)); the rate
 *       limits bound |log T_{t+1} - log T_t| and |theta_{t+1} - theta_t|.
 *   R14 scheduling priority: E[dH_s] is an exponential moving average of
 *       max(0, dH_s); C_s, M_s, L_s are kept tokens, context length and a
 *       caller urgency (Section 3.1 names them without formulas).
 *   R16 top-k estimators: K is the first k tokens by (y desc, token id asc);
 *       the tail mass is summed over the complement of K.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* Error bits; the values are part of the library's documented interface
 * and are restated (not shared) here. */
#define ORC_ERR_BAD_PAGE      0x1u
#define ORC_ERR_BAD_CTX       0x2u
#define ORC_ERR_NONFINITE     0x4u
#define ORC_ERR_ALL_NEG_INF   0x8u
#define ORC_ERR_BAD_TEMP      0x10u

int oracle_num_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* ------------------------------------------------------------------------ */
/* Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11, Section 3.3): a 4-word
 * counter, a 2-word key, ten rounds.  Each round multiplies words 0 and 2 by
 * the two round multipliers, keeps the 64-bit products, and forms the new
 * counter from the high halves xored with the other words and the round key
 * and the low halves; the key is bumped by the two Weyl constants between
 * rounds. */
static const uint32_t PHILOX_MUL0 = 0xD2511F53u;
static const uint32_t PHILOX_MUL1 = 0xCD9E8D57u;
static const uint32_t PHILOX_WEYL0 = 0x9E3779B9u;
static const uint32_t PHILOX_WEYL1 = 0xBB67AE85u;

void oracle_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
    uint32_t x0 = ctr[0], x1 = ctr[1], x2 = ctr[2], x3 = ctr[3];
    uint32_t k0 = key[0], k1 = key[1];
    for (int round = 0; round < 10; ++round) {
        uint64_t prod0 = (uint64_t)PHILOX_MUL0 * (uint64_t)x0;
        uint64_t prod1 = (uint64_t)PHILOX_MUL1 * (uint64_t)x2;
        uint32_t hi0 = (uint32_t)(prod0 >> 32), lo0 = (uint32_t)prod0;
        uint32_t hi1 = (uint32_t)(prod1 >> 32), lo1 = (uint32_t)prod1;
        uint32_t y0 = hi1 ^ x1 ^ k0;
        uint32_t y1 = lo1;
        uint32_t y2 = hi0 ^ x3 ^ k1;
        uint32_t y3 = lo0;
        x0 = y0; x1 = y1; x2 = y2; x3 = y3;
        k0 += PHILOX_WEYL0;
        k1 += PHILOX_WEYL1;
    }
    out[0] = x0; out[1] = x1; out[2] = x2; out[3] = x3;
}

/* The 32-bit random word that belongs to token x of row b:
 *   counter = (x / 4, b, lo32(offset), hi32(offset)), key = (lo32(seed), hi32(seed)),
 *   word    = output[x mod 4]. */
static uint32_t token_word(uint64_t seed, uint64_t offset, int64_t b, int64_t x) {
    uint32_t ctr[4] = {(uint32_t)(x >> 2), (uint32_t)b, (uint32_t)offset, (uint32_t)(offset >> 32)};
    uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
    uint32_t out[4];
    oracle_philox4x32_10(ctr, key, out);
    return out[x & 3];
}

/* Uniform in (0,1) from the low 23 bits of the word: u = (2j + 1) / 2^24. */
static double word_to_uniform(uint32_t w) {
    uint32_t j = w & 0x7FFFFFu;
    return ((double)(2u * j + 1u)) / 16777216.0;
}

void oracle_uniforms(uint64_t seed, uint64_t offset, int64_t b, int64_t x0, int64_t n, double *u) {
    for (int64_t i = 0; i < n; ++i) u[i] = word_to_uniform(token_word(seed, offset, b, x0 + i));
}

void oracle_words(const uint32_t *ctr, const uint32_t *key, int64_t n, uint32_t *out) {
    for (int64_t i = 0; i < n; ++i) oracle_philox4x32_10(ctr + 4 * i, key + 2 * i, out + 4 * i);
}

/* Gumbel-max key of token x: y_x + G_x with G_x = -log(-log u_x)
 * (argmax of the keys is a draw from softmax(y)). */
static double gumbel_key(double y, uint64_t seed, uint64_t offset, int64_t b, int64_t x) {
    double u = word_to_uniform(token_word(seed, offset, b, x));
    return y - log(-log(u));
}

/* Key of one token (used by tests to measure how far a disagreeing pick is
 * from the oracle's).  Returns -inf for a -inf logit. */
double oracle_sample_key(const float *logits_row, double T, uint64_t seed, uint64_t offset,
                         int64_t b, int64_t x) {
    double z = (double)logits_row[x];
    if (isinf(z) && z < 0) return -INFINITY;
    return gumbel_key(z / T, seed, offset, b, x);
}

/* ------------------------------------------------------------------------ */
/* Controller parameters (restated from the library header). */
typedef struct {
    double eta;        /* gain eta of the temperature law (Section 3.3) */
    double sign;       /* sigma in {-1, +1}; reading R1 */
    double T_min, T_max;
    double eps_H;      /* estimator error bound epsilon_H (Section 3.3) */
    double H_min;      /* entropy floor for pruning decisions (Section 5) */
    double theta_user; /* user threshold theta_t before the safety floor */
    double theta_hi;   /* scale of theta_max(H) */
    double T_cal;      /* global calibration temperature (Section 5; reading R13) */
    double rho_T;      /* bound on |log T_{t+1} - log T_t| per step, 0 = none (Section 5) */
    double dtheta;     /* bound on |theta_{t+1} - theta_t| per step, 0 = none (Section 5) */
} oracle_ctrl;

/*
 * One decode step's entropy, entropic time, temperature, threshold and sample.
 *
 *  H_t       = -sum_x p(x) log p(x),  p = softmax(z / T_t)       (Section 2.1)
 *  dH_t      = H_{t-1} - H_t,  tau += max(0, dH_t)               (Section 2, entropic time)
 *  T_{t+1}   = clip(T_t exp(sigma eta (H_t - H*)), T_min, T_max) (Section 3.3, reading R1)
 *  theta_{t+1} = min(theta_user, theta_max(max(H_t - eps_H, H_min)))
 *              (conservative-pruning floor, Section 3.2, and entropy floor, Section 5)
 *  theta_max(H) = theta_hi * max(0, 1 - H / log V)               (reading R6)
 *  tok       = argmax_x  z_x/T_t - log(-log u_x)                 (Gumbel-max draw from p)
 *  surprisal = -log p(tok)
 * Guards of Section 5 (reading R13): the logits are recalibrated by T_cal
 * before everything above (p from z / (T_cal T_t)); the new temperature is
 * kept within a factor e^{rho_T} of T_t before the [T_min, T_max] clip; the
 * new threshold within dtheta of the previous one, theta_prev[b] (a finite
 * previous threshold only; 0 turns either bound off).
 *
 * Outputs are double.  margin[b] = best key minus second-best key.  Rows with
 * a NaN or +inf logit, with every logit -inf, or with a temperature that is
 * not a positive finite number, set an error bit and return
 * H = NaN, tok = -1, T_out = T_in, theta_next = 0 (prune nothing), tau unchanged.
 */
void oracle_entropy_temp_sample(const float *logits, int B, int64_t V, int64_t ld,
                                const float *T_in, const float *H_prev, const float *tau_in,
                                const float *H_target, const oracle_ctrl *cp,
                                uint64_t seed, uint64_t offset, const float *theta_prev,
                                int32_t *tok, double *H, double *T_out, double *dH,
                                double *tau_out, double *theta_next, double *surprisal,
                                double *margin, uint32_t *err) {
    const double logV = log((double)V);
#pragma omp parallel for schedule(dynamic, 1)
    for (int b = 0; b < B; ++b) {
        const float *z = logits + (int64_t)b * ld;
        const double Tt = (double)T_in[b];
        const double T = Tt * cp->T_cal;          /* calibrated logits at temperature T_t */
        uint32_t e = (T > 0.0 && !isinf(T)) ? 0u : ORC_ERR_BAD_TEMP;
        double m = -INFINITY;
        for (int64_t x = 0; x < V && !e; ++x) {
            double zx = (double)z[x];
            if (isnan(zx) || (isinf(zx) && zx > 0)) e |= ORC_ERR_NONFINITE;
            else if (zx / T > m) m = zx / T;
        }
        if (!e && isinf(m)) e |= ORC_ERR_ALL_NEG_INF;
        err[b] = e;
        if (e) {
            tok[b] = -1; H[b] = NAN; dH[b] = NAN; T_out[b] = Tt;
            tau_out[b] = (double)tau_in[b]; theta_next[b] = 0.0;
            surprisal[b] = NAN; margin[b] = NAN;
            continue;
        }
        /* pass 1: normaliser */
        double S = 0.0;
        for (int64_t x = 0; x < V; ++x) {
            double y = (double)z[x] / T;
            S += exp(y - m);
        }
        /* pass 2: entropy by its definition, 0 log 0 := 0 */
        double h = 0.0;
        for (int64_t x = 0; x < V; ++x) {
            double p = exp((double)z[x] / T - m) / S;
            if (p > 0.0) h -= p * log(p);
        }
        /* pass 3: Gumbel-max sample; ties go to the lowest token id */
        double best = -INFINITY, second = -INFINITY;
        int64_t arg = -1;
        for (int64_t x = 0; x < V; ++x) {
            double zx = (double)z[x];
            if (isinf(zx)) continue; /* -inf logits are never drawn */
            double k = gumbel_key(zx / T, seed, offset, b, x);
            if (k > best) { second = best; best = k; arg = x; }
            else if (k > second) second = k;
        }
        H[b] = h;
        tok[b] = (int32_t)arg;
        margin[b] = best - second;
        surprisal[b] = -(((double)z[arg] / T - m) - log(S));
        dH[b] = (double)H_prev[b] - h;
        tau_out[b] = (double)tau_in[b] + fmax(0.0, dH[b]);
        double Tn = Tt * exp(cp->sign * cp->eta * (h - (double)H_target[b]));
        if (cp->rho_T > 0.0) Tn = fmin(Tt * exp(cp->rho_T), fmax(Tt * exp(-cp->rho_T), Tn));
        T_out[b] = fmin(cp->T_max, fmax(cp->T_min, Tn));
        double Heff = fmax(h - cp->eps_H, cp->H_min);
        double tmax = (V > 1) ? cp->theta_hi * fmax(0.0, 1.0 - Heff / logV) : cp->theta_hi;
        double th = fmin(cp->theta_user, tmax);
        if (cp->dtheta > 0.0 && theta_prev && isfinite((double)theta_prev[b])) {
            const double tp = (double)theta_prev[b];
            th = fmin(tp + cp->dtheta, fmax(tp - cp->dtheta, th));
        }
        theta_next[b] = th;
    }
}

/* Entropy of softmax(z / T) for one row, by definition (used by pins). */
double oracle_entropy_row(const float *z, int64_t V, double T) {
    double m = -INFINITY;
    for (int64_t x = 0; x < V; ++x) if ((double)z[x] / T > m) m = (double)z[x] / T;
    double S = 0.0;
    for (int64_t x = 0; x < V; ++x) S += exp((double)z[x] / T - m);
    double h = 0.0;
    for (int64_t x = 0; x < V; ++x) {
        double p = exp((double)z[x] / T - m) / S;
        if (p > 0.0) h -= p * log(p);
    }
    return h;
}

/* ------------------------------------------------------------------------ */
/* Entropy-aware scheduling priority and admission (Section 3.1, reading R14).
 *
 *   E[dH_s] <- lambda E[dH_s] + (1 - lambda) max(0, dH_s)   (the expected
 *              irreversible entropy reduction, an exponential moving average of
 *              the reductions that entropic time counts; a NaN dH leaves it)
 *   C_s = kept tokens per kv head (attention work of the step),
 *   M_s = context length (KV memory), L_s = caller-given urgency,
 *   pi(s) = E[dH_s] / max(alpha C_s + beta M_s + gamma L_s, den_min)
 * and the `budget` sequences of highest pi are admitted (ties to the lower
 * index; a NaN priority ranks below every number).  kept_cnt, ctx_lens and
 * urgency may be NULL (the term is 0). */
typedef struct {
    double lambda, alpha, beta, gamma, den_min;
} oracle_sched;

typedef struct { double pi; int idx; } sched_item;

static int sched_cmp(const void *pa, const void *pb) {
    const sched_item *a = (const sched_item *)pa, *b = (const sched_item *)pb;
    const int na = isnan(a->pi), nb = isnan(b->pi);
    if (na != nb) return na - nb;               /* NaN after every number */
    if (!na) {
        if (a->pi > b->pi) return -1;
        if (a->pi < b->pi) return 1;
    }
    return (a->idx > b->idx) - (a->idx < b->idx);
}

void oracle_schedule(const float *dH, const float *ema_in, const int32_t *kept_cnt, int Hkv, int P,
                     const int32_t *ctx_lens, const float *urgency, const oracle_sched *sp, int B,
                     int budget, double *ema_out, double *priority, uint8_t *admit) {
    sched_item *order = (sched_item *)malloc(sizeof(sched_item) * (size_t)(B > 0 ? B : 1));
    for (int s = 0; s < B; ++s) {
        const double d = (double)dH[s];
        double e = (double)ema_in[s];
        if (!isnan(d)) e = sp->lambda * e + (1.0 - sp->lambda) * fmax(0.0, d);
        double C = 0.0;
        if (kept_cnt) {
            for (int h = 0; h < Hkv; ++h) C += (double)kept_cnt[(int64_t)s * Hkv + h] * P;
            C /= Hkv;
        }
        const double M = ctx_lens ? (double)ctx_lens[s] : 0.0;
        const double L = urgency ? (double)urgency[s] : 0.0;
        const double den = fmax(sp->alpha * C + sp->beta * M + sp->gamma * L, sp->den_min);
        ema_out[s] = e;
        priority[s] = e / den;
        order[s].pi = priority[s];
        order[s].idx = s;
        admit[s] = 0;
    }
    qsort(order, (size_t)B, sizeof(sched_item), sched_cmp);
    const int n = budget < B ? (budget > 0 ? budget : 0) : B;
    for (int r = 0; r < n; ++r) admit[order[r].idx] = 1;
    free(order);
}

/* ------------------------------------------------------------------------ */
/* Top-k entropy estimators (Section 2.1, "Top-k entropy approximation" and
 * "Tail-corrected estimator").
 *
 * With y = z / T_t, p = softmax(y) and K the first k_eff = min(k, V) tokens
 * ordered by (y descending, token id ascending):
 *   p~(x)   = p(x) / sum_{y in K} p(y) on K            (truncated distribution)
 *   H~      = -sum_{x in K} p~(x) log p~(x)            (0 log 0 := 0)
 *   m       = sum_{x in K} p(x),   m_bar = 1 - m = sum_{x not in K} p(x)
 *   H^      = H~ + h(m_bar) + m_bar log(V - k_eff)     (h: binary entropy;
 *                                                       the last term is 0 when k_eff = V)
 * tail_mass = m_bar, summed over the tail itself so that a small tail keeps
 * its relative precision.  Rows with a NaN or +inf logit, with every logit
 * -inf, or with a temperature that is not a positive finite number set their
 * error bit and return NaN. */
typedef struct { double y; int64_t idx; } topk_item;

static int topk_cmp(const void *pa, const void *pb) {
    const topk_item *a = (const topk_item *)pa, *b = (const topk_item *)pb;
    if (a->y > b->y) return -1;
    if (a->y < b->y) return 1;
    return (a->idx > b->idx) - (a->idx < b->idx);
}

void oracle_topk_entropy(const float *logits, int B, int64_t V, int64_t ld, const float *T_in,
                         int64_t k, double *H_tilde, double *H_hat, double *tail_mass,
                         uint32_t *err) {
#pragma omp parallel for schedule(dynamic, 1)
    for (int b = 0; b < B; ++b) {
        const float *z = logits + (int64_t)b * ld;
        const double T = (double)T_in[b];
        uint32_t e = (T > 0.0 && !isinf(T)) ? 0u : ORC_ERR_BAD_TEMP;
        double M = -INFINITY;
        for (int64_t x = 0; x < V && !e; ++x) {
            double zx = (double)z[x];
            if (isnan(zx) || (isinf(zx) && zx > 0)) e |= ORC_ERR_NONFINITE;
            else if (zx / T > M) M = zx / T;
        }
        if (!e && isinf(M)) e |= ORC_ERR_ALL_NEG_INF;
        err[b] = e;
        if (e) { H_tilde[b] = NAN; H_hat[b] = NAN; tail_mass[b] = NAN; continue; }
        topk_item *it = (topk_item *)malloc(sizeof(topk_item) * (size_t)V);
        for (int64_t x = 0; x < V; ++x) { it[x].y = (double)z[x] / T; it[x].idx = x; }
        qsort(it, (size_t)V, sizeof(topk_item), topk_cmp);
        const int64_t ke = k < V ? k : V;
        double ZK = 0.0, Zt = 0.0;
        for (int64_t r = 0; r < V; ++r) {
            double w = exp(it[r].y - M);
            if (r < ke) ZK += w; else Zt += w;
        }
        double h = 0.0;
        for (int64_t r = 0; r < ke; ++r) {
            double pt = exp(it[r].y - M) / ZK;
            if (pt > 0.0) h -= pt * log(pt);
        }
        const double mb = Zt / (ZK + Zt);
        double hb = 0.0;
        if (mb > 0.0 && mb < 1.0) hb = -mb * log(mb) - (1.0 - mb) * log1p(-mb);
        H_tilde[b] = h;
        tail_mass[b] = mb;
        H_hat[b] = h + hb + (ke < V ? mb * log((double)(V - ke)) : 0.0);
        free(it);
    }
}

/* ------------------------------------------------------------------------ */
/* Paged KV cache helpers.  k_cache / v_cache are bf16 bit patterns laid out
 * [num_pages][Hkv][P][D]; block_table is [B][max_blocks]. */

static double bf16_to_double(uint16_t bits) {
    uint32_t w = (uint32_t)bits << 16;
    float f;
    memcpy(&f, &w, sizeof f);
    return (double)f;
}

/* Returns the error bits of sequence b (bad context length, bad page id). */
static uint32_t seq_check(const int32_t *block_table, const int32_t *ctx_lens, int b,
                          int P, int max_blocks, int64_t num_pages) {
    int L = ctx_lens[b];
    if (L < 0 || (int64_t)L > (int64_t)max_blocks * P) return ORC_ERR_BAD_CTX;
    int nb = (L + P - 1) / P;
    for (int j = 0; j < nb; ++j) {
        int32_t pg = block_table[(int64_t)b * max_blocks + j];
        if (pg < 0 || (int64_t)pg >= num_pages) return ORC_ERR_BAD_PAGE;
    }
    return 0;
}

/* Scaled dot products x_i = scale * q_h . k_i for every token i < L of
 * sequence b, query head h. */
static void head_logits(const uint16_t *q, const uint16_t *k_cache, const int32_t *block_table,
                        int b, int h, int L, int Hq, int Hkv, int D, int P, int max_blocks,
                        double scale, double *x) {
    int g = Hq / Hkv, kvh = h / g;
    const uint16_t *qh = q + ((int64_t)b * Hq + h) * D;
    for (int i = 0; i < L; ++i) {
        int64_t page = block_table[(int64_t)b * max_blocks + i / P];
        const uint16_t *kr = k_cache + (((page * Hkv + kvh) * P) + (i % P)) * (int64_t)D;
        double s = 0.0;
        for (int d = 0; d < D; ++d) s += bf16_to_double(qh[d]) * bf16_to_double(kr[d]);
        x[i] = scale * s;
    }
}

typedef struct { double score; int idx; } rank_item;

/* (score desc, index asc) */
static int rank_cmp(const void *pa, const void *pb) {
    const rank_item *a = (const rank_item *)pa, *b = (const rank_item *)pb;
    if (a->score > b->score) return -1;
    if (a->score < b->score) return 1;
    return (a->idx > b->idx) - (a->idx < b->idx);
}

/*
 * Entropic block scores and keep set (Section 3.2 with readings R4-R7).
 *
 * For each query head h and token i < L_b:  a_i = softmax_i(x_i) over all
 * L_b tokens;  I_b^(h) = sum_{i in block} a_i * I_i with I_i = -log a_i
 * (score_mode 0, A), surp[page(i) * P + i mod P] (1, E: the stored token
 * surprisal, paged like the keys: [num_pages][P]) or 1 (2, M);
 * normalised  Ibar_b^(h) = n_b I_b^(h) / sum_b' I_b'^(h)  (1 when the sum is 0);
 * group score Ibar_b = max over the heads of the kv group.
 * keep_b  iff  Ibar_b >= theta[b]  or  b is among the first min(B_min, n_b)
 * blocks ordered by (Ibar desc, b asc).
 *
 * Outputs: keep_mask [B][Hkv][max_blocks] (0/1), kept_idx [B][Hkv][max_blocks]
 * (ascending, -1 padded), kept_cnt [B][Hkv], block_score [B][Hkv][max_blocks]
 * (Ibar, 0 padded), head_I [B][Hq][max_blocks] (raw I_b^(h)),
 * head_A [B][Hq][max_blocks] (block attention mass sum_{i in block} a_i) and
 * head_H [B][Hq] (attention entropy) -- the last three may be NULL.
 * A sequence with a bad page id or context length keeps nothing.
 */
void oracle_score_prune(const uint16_t *q, const uint16_t *k_cache, const int32_t *block_table,
                        const int32_t *ctx_lens, int B, int Hq, int Hkv, int D, int P,
                        int max_blocks, int64_t num_pages, double scale,
                        const float *theta, int B_min, int score_mode, const float *surp,
                        uint8_t *keep_mask, int32_t *kept_idx, int32_t *kept_cnt,
                        double *block_score, double *head_I, double *head_A, double *head_H,
                        uint32_t *err) {
    const int g = Hq / Hkv;
    for (int b = 0; b < B; ++b) err[b] = seq_check(block_table, ctx_lens, b, P, max_blocks, num_pages);
#pragma omp parallel for collapse(2) schedule(dynamic, 1)
    for (int b = 0; b < B; ++b) {
        for (int kvh = 0; kvh < Hkv; ++kvh) {
            int64_t seg = (int64_t)b * Hkv + kvh;
            uint8_t *km = keep_mask + seg * max_blocks;
            int32_t *ki = kept_idx + seg * max_blocks;
            double *bs = block_score + seg * max_blocks;
            for (int j = 0; j < max_blocks; ++j) { km[j] = 0; ki[j] = -1; bs[j] = 0.0; }
            kept_cnt[seg] = 0;
            for (int hh = 0; hh < g; ++hh)
                for (int j = 0; j < max_blocks; ++j) {
                    int64_t o = ((int64_t)b * Hq + kvh * g + hh) * max_blocks + j;
                    if (head_I) head_I[o] = 0.0;
                    if (head_A) head_A[o] = 0.0;
                }
            if (head_H) for (int hh = 0; hh < g; ++hh) head_H[(int64_t)b * Hq + kvh * g + hh] = 0.0;
            int L = ctx_lens[b];
            if (err[b] || L == 0) continue;
            int nb = (L + P - 1) / P;
            double *x = (double *)malloc(sizeof(double) * (size_t)L);
            double *Ih = (double *)malloc(sizeof(double) * (size_t)nb);
            double *Ah = (double *)malloc(sizeof(double) * (size_t)nb);
            double *score = (double *)malloc(sizeof(double) * (size_t)nb);
            for (int j = 0; j < nb; ++j) score[j] = -INFINITY;
            for (int hh = 0; hh < g; ++hh) {
                int h = kvh * g + hh;
                head_logits(q, k_cache, block_table, b, h, L, Hq, Hkv, D, P, max_blocks, scale, x);
                double M = -INFINITY;
                for (int i = 0; i < L; ++i) if (x[i] > M) M = x[i];
                double Z = 0.0;
                for (int i = 0; i < L; ++i) Z += exp(x[i] - M);
                double total = 0.0;
                for (int j = 0; j < nb; ++j) {
                    double s = 0.0, mass = 0.0;
                    int i1 = (j + 1) * P < L ? (j + 1) * P : L;
                    for (int i = j * P; i < i1; ++i) {
                        double a = exp(x[i] - M) / Z;
                        mass += a;
                        if (score_mode == 1) {
                            int64_t page = block_table[(int64_t)b * max_blocks + j];
                            s += a * (double)surp[page * P + (i - j * P)];
                        } else if (score_mode == 2) {
                            s += a;
                        } else if (a > 0.0) {
                            s += a * (-log(a));
                        }
                    }
                    Ih[j] = s;
                    Ah[j] = mass;
                    total += s;
                }
                for (int j = 0; j < nb; ++j) {
                    double nrm = total > 0.0 ? (double)nb * Ih[j] / total : 1.0;
                    if (nrm > score[j]) score[j] = nrm;
                    if (head_I) head_I[((int64_t)b * Hq + h) * max_blocks + j] = Ih[j];
                    if (head_A) head_A[((int64_t)b * Hq + h) * max_blocks + j] = Ah[j];
                }
                if (head_H) head_H[(int64_t)b * Hq + h] = total;
            }
            /* order blocks by (score desc, index asc) with a library sort and
             * mark the first min(B_min, n_b) of that order */
            int kmin = B_min < nb ? B_min : nb;
            if (kmin < 0) kmin = 0;
            uint8_t *taken = (uint8_t *)calloc((size_t)nb, 1);
            rank_item *order = (rank_item *)malloc(sizeof(rank_item) * (size_t)nb);
            for (int j = 0; j < nb; ++j) { order[j].score = score[j]; order[j].idx = j; }
            qsort(order, (size_t)nb, sizeof(rank_item), rank_cmp);
            for (int r = 0; r < kmin; ++r) taken[order[r].idx] = 1;
            free(order);
            double th = (double)theta[b];
            int cnt = 0;
            for (int j = 0; j < nb; ++j) {
                int keep = taken[j] || score[j] >= th;
                km[j] = (uint8_t)keep;
                bs[j] = score[j];
                if (keep) ki[cnt++] = j;
            }
            kept_cnt[seg] = cnt;
            free(taken); free(score); free(Ah); free(Ih); free(x);
        }
    }
}

/*
 * Paged GQA decode attention restricted to the kept blocks (Section 3.2,
 * reading R8): out_h = sum_{i kept} softmax_kept(x_i) v_i, with the softmax
 * taken over the kept tokens only.  keep_mask == NULL means every block is
 * kept (dense decode).  A sequence with no kept token, a bad page id or a bad
 * context length gets a zero output.  out is [B][Hq][D] double.
 */
void oracle_paged_attention(const uint16_t *q, const uint16_t *k_cache, const uint16_t *v_cache,
                            const int32_t *block_table, const int32_t *ctx_lens,
                            int B, int Hq, int Hkv, int D, int P, int max_blocks,
                            int64_t num_pages, double scale, const uint8_t *keep_mask,
                            double *out, uint32_t *err) {
    const int g = Hq / Hkv;
    for (int b = 0; b < B; ++b) err[b] = seq_check(block_table, ctx_lens, b, P, max_blocks, num_pages);
#pragma omp parallel for collapse(2) schedule(dynamic, 1)
    for (int b = 0; b < B; ++b) {
        for (int h = 0; h < Hq; ++h) {
            double *o = out + ((int64_t)b * Hq + h) * D;
            for (int d = 0; d < D; ++d) o[d] = 0.0;
            int L = ctx_lens[b];
            if (err[b] || L == 0) continue;
            int kvh = h / g;
            double *x = (double *)malloc(sizeof(double) * (size_t)L);
            head_logits(q, k_cache, block_table, b, h, L, Hq, Hkv, D, P, max_blocks, scale, x);
            const uint8_t *km = keep_mask ? keep_mask + ((int64_t)b * Hkv + kvh) * max_blocks : NULL;
            double M = -INFINITY;
            for (int i = 0; i < L; ++i) if ((!km || km[i / P]) && x[i] > M) M = x[i];
            if (isinf(M)) { free(x); continue; } /* nothing kept */
            double Z = 0.0;
            for (int i = 0; i < L; ++i) if (!km || km[i / P]) Z += exp(x[i] - M);
            for (int i = 0; i < L; ++i) {
                if (km && !km[i / P]) continue;
                double a = exp(x[i] - M) / Z;
                int64_t page = block_table[(int64_t)b * max_blocks + i / P];
                const uint16_t *vr = v_cache + (((page * Hkv + kvh) * P) + (i % P)) * (int64_t)D;
                for (int d = 0; d < D; ++d) o[d] += a * bf16_to_double(vr[d]);
            }
            free(x);
        }
    }
}
