/*
 * eti.h -- C ABI of libeti, the GB300 (sm_103a) kernels of the entropic-time
 * batched decode step (Kiruluta, "Entropic-Time Inference: Self-Organizing
 * Large Language Model Decoding Beyond Attention", arXiv 2603.03310).
 *
 * The step has two halves:
 *   (a) per sequence: softmax and Shannon entropy H_t of the vocabulary
 *       logits at the current temperature T_t (Section 2.1), the entropy
 *       flow dH_t and entropic time tau (Section 2), the next temperature
 *       (Section 3.3), the next pruning threshold (Section 3.2,
 *       "Conservative pruning", and Section 5, entropy floor) and a token
 *       drawn from p_t;
 *   (b) per sequence and kv head: entropic scores of the paged KV blocks
 *       (Section 3.2, I_b), the keep set B_t = {b : I_b >= theta_t} with the
 *       minimum block budget B_min (Section 3.2), and GQA paged decode
 *       attention restricted to B_t.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - Every tensor argument is a DEVICE pointer owned by the caller, row-major
 *    and contiguous unless a leading dimension is given; outputs are
 *    preallocated by the caller.  bf16 data is passed as uint16_t bit
 *    patterns (eti_bf16).  Small parameter structs are HOST pointers and are
 *    read before the call returns.
 *  - `stream` is a cudaStream_t (NULL = legacy default stream).  Calls only
 *    enqueue work: they never synchronise, never allocate device memory and
 *    keep no state between calls.  Scratch comes from the caller's `ws`
 *    buffer, sized by the matching *_workspace_size() function.
 *  - Return value: ETI_OK or a negative ETI_ERR_* status for argument errors
 *    detected on the host (nothing is enqueued then) or a failed launch.
 *  - Problems found in the DATA on the device never trap: each call writes
 *    one word of ETI_ERRF_* bits per sequence into `err_flags` (uint32 [B],
 *    overwritten, 0 = fine) and gives that sequence a defined fallback
 *    result, documented per call.
 *  - Supported shapes: head_dim D in {64, 128}; page size P in {16, 32};
 *    Hq % Hkv == 0 with group size g = Hq / Hkv <= 8; 1 <= max_blocks <= 32768;
 *    B <= 65535 (entropy/sample) or 8192 (attention calls); 1 <= V.
 *    Attention calls also need B * Hkv * max_blocks <= 2^30 and
 *    num_pages * Hkv * P < 2^31 (block counts and cache rows are 32-bit
 *    indices on the device); larger shapes return ETI_ERR_UNSUPPORTED.
 *    q, k_cache, v_cache, token_scores and the decode output must be 16-byte
 *    aligned.
 *
 * Layouts
 *  - q          bf16  [B][Hq][D]
 *  - k_cache    bf16  [num_pages][Hkv][P][D]   (one (page, kv head) chunk is
 *    v_cache    bf16  [num_pages][Hkv][P][D]    P*D*2 contiguous bytes)
 *  - block_table int32 [B][max_blocks]: physical page of logical block j of
 *    sequence b; only entries j < ceil(ctx_lens[b] / P) are read.
 *  - ctx_lens   int32 [B]: tokens of sequence b (0 allowed).
 *  - keep_mask  uint8 [B][Hkv][max_blocks]; kept_idx int32 [B][Hkv][max_blocks]
 *    (kept block indices ascending, -1 after kept_cnt); kept_cnt int32 [B][Hkv].
 *  - token_scores fp32 [B][Hkv][max_blocks][P][g]: x_i = scale * q_h . k_i
 *    for every token slot (-inf past the sequence end).
 *  - kept_norm  fp32 [B][Hq][2]: (max, sum of exp(x - max)) of the softmax
 *    over the kept tokens of each query head.
 */
#ifndef ETI_H_
#define ETI_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef uint16_t eti_bf16;

/* status codes */
#define ETI_OK               0
#define ETI_ERR_NULL        (-1)  /* a required pointer is NULL */
#define ETI_ERR_SHAPE       (-2)  /* a size is out of range or inconsistent */
#define ETI_ERR_UNSUPPORTED (-3)  /* a valid shape this library does not implement */
#define ETI_ERR_WORKSPACE   (-4)  /* ws is NULL or smaller than *_workspace_size() */
#define ETI_ERR_CUDA        (-5)  /* a kernel launch failed (cudaGetLastError) */
#define ETI_ERR_TIMEOUT     (-6)  /* reserved: no call returns it.  Calls never wait on the
                                     host; a device-side wait that gives up is reported per
                                     sequence by ETI_ERRF_TIMEOUT in err_flags */
#define ETI_ERR_TOO_LARGE   (-7)  /* the problem needs more than the fixed scratch of
                                     eti_entropy_temp_sample_noalloc */
#define ETI_ERR_ALIGN       (-8)  /* a bf16 tensor is not 16-byte aligned */

/* per-sequence data error bits written to err_flags */
#define ETI_ERRF_BAD_PAGE     0x1u  /* a block_table entry is outside [0, num_pages) */
#define ETI_ERRF_BAD_CTX      0x2u  /* ctx_len < 0 or > max_blocks * P */
#define ETI_ERRF_NONFINITE    0x4u  /* a logit is NaN or +inf */
#define ETI_ERRF_ALL_NEG_INF  0x8u  /* every logit of the row is -inf */
#define ETI_ERRF_BAD_TEMP     0x10u /* T_in is not a positive finite number */
#define ETI_ERRF_TIMEOUT      0x20u /* a device-side wait for a tile copy gave up (the
                                       sequence's results are not valid) */
#define ETI_ERRF_DRAIN        0x40u /* with TIMEOUT: after the wait gave up, a tile copy
                                       already issued did not land within the drain
                                       limit either, so it may still write shared
                                       memory after its CTA exited: treat the device
                                       as suspect, not only the sequence */

/*
 * Controller parameters (Section 3.3 temperature law, Section 3.2 safety
 * floor, Section 5 guards).  The paper gives no values; eti_ctrl_defaults()
 * fills the defaults this library documents.
 *   eta         gain of the temperature law                       (default 0.1)
 *   sign        -1: T' = T exp(eta (H* - H)), which restores H toward H*
 *               because H grows with T; +1: the law exactly as printed in
 *               Section 3.3, which is positive feedback          (default -1)
 *   T_min,T_max clip range of the temperature               (0.05, 5.0)
 *   eps_H       bound on the entropy-estimate error, subtracted before the
 *               threshold floor (Section 3.2)                     (0)
 *   H_min       entropy floor for pruning decisions (Section 5)   (0)
 *   theta_user  threshold before the safety floor                 (+inf)
 *   theta_hi    scale of theta_max(H) = theta_hi * max(0, 1 - H / log V) (1)
 *   T_cal       global calibration temperature: the logits are read as
 *               z / T_cal before everything else (Section 5)       (1)
 *   rho_T       bound on |log T_out - log T_in| per step, applied before
 *               the [T_min, T_max] clip; 0 = none (Section 5)        (0)
 *   dtheta      bound on |theta_next - theta_prev| per step; when > 0,
 *               theta_next is read first as the previous threshold (in
 *               place, like tau; a non-finite previous value is not
 *               bounded); 0 = none (Section 5)                        (0)
 */
typedef struct {
    float eta;
    float sign;
    float T_min;
    float T_max;
    float eps_H;
    float H_min;
    float theta_user;
    float theta_hi;
    float T_cal;
    float rho_T;
    float dtheta;
} eti_ctrl_params;

void eti_ctrl_defaults(eti_ctrl_params* p);

/*
 * eti_entropy_temp_sample -- half (a) of the step, one fused pass per row.
 *
 * For each sequence b, with y = z / T_in[b] over the first V entries of row
 * b of `logits` (fp32, row stride ld >= V elements):
 *   H[b]       = -sum_x p(x) log p(x),  p = softmax(y)          (Section 2.1)
 *   dH[b]      = H_prev[b] - H[b]                                (Section 2)
 *   tau[b]    += max(0, dH[b])         (entropic time, in place; Section 2)
 *   T_out[b]   = clip(T_in[b] exp(sign eta (H[b] - H_target[b])), T_min, T_max)
 *                                                                (Section 3.3)
 *   (with the Section 5 guards of eti_ctrl_params: y = z / (T_cal T_in[b]),
 *   the rho_T bound on the step of T, the dtheta bound on theta_next)
 *   theta_next[b] = min(theta_user, theta_hi max(0, 1 - max(H - eps_H, H_min) / log V))
 *                  (threshold floor of Section 3.2 with the Section 5 floor;
 *                   theta_hi when V == 1)
 *   tok[b]     = argmax_x y_x - log(-log u_x): a draw from p by the Gumbel-max
 *                rule, u_x from Philox4x32-10 with counter
 *                (x / 4, b, lo32(offset), hi32(offset)), key (lo32(seed),
 *                hi32(seed)), word x mod 4, u = (2 (word & 0x7FFFFF) + 1) / 2^24;
 *                ties go to the lowest token id; -inf logits are never drawn
 *   tok_surprisal[b] = -log p(tok)  (also written to surp_store, see above)
 * H, dH, T_out, theta_next, tok_surprisal: fp32 [B]; tok: int32 [B];
 * dH, theta_next, tok_surprisal may be NULL.  T_in, H_prev, H_target: fp32
 * [B].  T_out may alias T_in.
 * Row errors (NaN/+inf logit, all -inf, bad T_in) give tok = -1, H = dH =
 * surprisal = NaN, T_out = T_in, theta_next = 0 (prune nothing), tau unchanged.
 * The row is computed in fp32 on z * log2(e) / (T_cal T_in): a row where that
 * product overflows (|z| / (T_cal T_in) above about 2.36e38, or T_cal T_in
 * below about 4.2e-39) is reported as ETI_ERRF_NONFINITE as well.
 * offset_dev: NULL, or a device uint64 that replaces `offset`: the call reads
 * the counter from it and, once every row is drawn, stores counter + 1 back,
 * so that a captured CUDA graph draws fresh numbers at every replay.  Calls
 * that share one offset_dev word must not overlap on the GPU.
 * Workspace: eti_entropy_temp_sample_workspace_size(B, V) bytes, 4-byte
 * aligned (row tickets and partial reductions of the row pieces; no initial
 * contents required: the call zeroes its tickets itself).
 */
size_t eti_entropy_temp_sample_workspace_size(int B, int V);

/*
 * Where eti_entropy_temp_sample records each drawn token's surprisal for
 * score mode E (the whole struct is nullable; it is a HOST pointer read
 * before the call returns, the arrays are device memory):
 *   store[slot_mapping[b]] = -log p(tok[b])
 * for every sequence with no error bit and 0 <= slot_mapping[b] < num_slots
 * (the slot of the position the new token takes in the caller's paged
 * layout: page * P + offset; a negative slot skips the sequence).
 */
typedef struct {
    float* store;                 /* fp32 [num_slots] */
    const int64_t* slot_mapping;  /* int64 [B] */
    int64_t num_slots;
} eti_surp_store;

int eti_entropy_temp_sample(const float* logits, int B, int V, int64_t ld,
                            const float* T_in, const float* H_prev, float* tau,
                            const float* H_target, const eti_ctrl_params* params,
                            uint64_t seed, uint64_t offset, uint64_t* offset_dev,
                            int32_t* tok, float* H, float* T_out,
                            float* dH, float* theta_next, float* tok_surprisal,
                            const eti_surp_store* surp_store,
                            uint32_t* err_flags, void* ws, size_t ws_bytes, void* stream);

/*
 * eti_entropy_temp_sample_noalloc -- the same computation, arguments and
 * results as eti_entropy_temp_sample, for callers that cannot allocate
 * device memory at all: code that is handed only its input and output
 * buffers by a host framework that owns every device allocation (a plugin
 * or callback with no workspace argument and no allocator to ask), or a
 * latency-critical host thread that must never enter the CUDA allocator.
 * The paper has no counterpart; this is a deployment convenience.
 *
 * Instead of a workspace, the call uses a fixed scratch array compiled into
 * this library (eti_entropy_temp_sample_noalloc_max_bytes() bytes, one copy
 * on every GPU that loads the library, kept until the process exits).  It
 * never calls cudaMalloc, cudaFree or any allocating routine.
 *  - The first call on a device looks up that array's device address
 *    (cudaGetSymbolAddress) with the device current, once per device (and
 *    again if the device's current context changes, e.g. after
 *    cudaDeviceReset); make that first call before any stream capture.
 *  - Every call on a device shares the one array and it keeps the previous
 *    call's contents; nothing in it needs to start at zero: each call first
 *    clears the row tickets it uses (a small kernel in the same stream), and
 *    every other entry it reads was written earlier by the same call.  Calls
 *    whose execution overlaps on the GPU (other streams, or several host
 *    threads) race on the array: serialise them.
 *  - A problem whose scratch (eti_entropy_temp_sample_workspace_size(B, V))
 *    exceeds the array returns ETI_ERR_TOO_LARGE and enqueues nothing; at
 *    152 SMs the limit is about 16,600 sequences, whatever V is.
 */
size_t eti_entropy_temp_sample_noalloc_max_bytes(void);

int eti_entropy_temp_sample_noalloc(const float* logits, int B, int V, int64_t ld,
                                    const float* T_in, const float* H_prev, float* tau,
                                    const float* H_target, const eti_ctrl_params* params,
                                    uint64_t seed, uint64_t offset, uint64_t* offset_dev,
                                    int32_t* tok, float* H, float* T_out,
                                    float* dH, float* theta_next, float* tok_surprisal,
                                    const eti_surp_store* surp_store,
                                    uint32_t* err_flags, void* stream);

/*
 * Entropy-aware scheduling (Section 3.1): the priority
 *   pi(s) = E[dH_s | S_t] / (alpha C_s + beta M_s + gamma L_s)
 * with (the paper names the terms without formulas):
 *   E[dH_s]  an exponential moving average of the irreversible entropy
 *            reduction max(0, dH_s) that entropic time counts:
 *            ema[s] <- lambda ema[s] + (1 - lambda) max(0, dH[s]) in place
 *            (a NaN dH, an error row, leaves it unchanged);
 *   C_s      attention work: kept tokens per kv head,
 *            sum_h kept_cnt[s][h] * P / Hkv (0 when kept_cnt is NULL);
 *   M_s      KV memory: ctx_lens[s] tokens (0 when NULL);
 *   L_s      urgency[s], the caller's latency risk (0 when NULL);
 * and the denominator floored at den_min.  The `budget` sequences of highest
 * priority are admitted: admit_mask[s] = 1 (ties to the lower index, a NaN
 * priority below every number; budget <= 0 admits none, >= B all).
 * Parameters (defaults from eti_sched_defaults): lambda 0.9, alpha 1e-3,
 * beta 1e-3 (per token), gamma 1, den_min 1e-6.  B <= 65535; one CTA.
 */
typedef struct {
    float lambda;
    float alpha;
    float beta;
    float gamma;
    float den_min;
} eti_sched_params;

void eti_sched_defaults(eti_sched_params* p);

int eti_schedule(const float* dH, float* ema, const int32_t* kept_cnt, int Hkv, int P,
                 const int32_t* ctx_lens, const float* urgency, const eti_sched_params* params,
                 int B, int budget, float* priority, uint8_t* admit_mask, void* stream);

/*
 * eti_topk_entropy -- the top-k entropy estimators of Section 2.1, for each
 * row b with y = z / T_in[b] over the first V entries of row b of `logits`
 * (fp32, row stride ld >= V), p = softmax(y) and K the first min(k, V) tokens
 * ordered by (y descending, token id ascending):
 *   H_tilde[b]   = -sum_{x in K} p~(x) log p~(x),  p~ = p / sum_K p
 *   tail_mass[b] = sum_{x not in K} p(x)            (= 1 - m_t; nullable)
 *   H_hat[b]     = H_tilde + h(tail) + tail log(V - k)   (tail-corrected;
 *                  the last term is 0 when k >= V; h: binary entropy)
 * err_flags as for eti_entropy_temp_sample (NONFINITE, ALL_NEG_INF,
 * BAD_TEMP; those rows get NaN).  k >= 1 (k > V is V).  No workspace; one
 * pass over the logits from HBM and three from L2.
 */
int eti_topk_entropy(const float* logits, int B, int V, int64_t ld, const float* T_in, int k,
                     float* H_tilde, float* H_hat, float* tail_mass, uint32_t* err_flags,
                     void* stream);

/*
 * Score modes: the reading of "the surprisal associated with the value
 * vector" I(v_i) in the block score of Section 3.2.
 *   ETI_SCORE_A  I(v_i) = -log a_i (attention as a distribution over the
 *                values; the block scores add up to the attention entropy)
 *   ETI_SCORE_E  I(v_i) = the stored surprisal -log p(x_i | x_<i) of the
 *                token at position i, recorded when it was generated; the
 *                store is fp32 [num_pages][P], paged like the keys (token i
 *                of sequence b at tok_surp[block_table[b][i / P] * P + i % P])
 *                and written by eti_entropy_temp_sample's surp_store output
 *   ETI_SCORE_M  I(v_i) = 1 (the block's attention mass)
 */
#define ETI_SCORE_A 0
#define ETI_SCORE_E 1
#define ETI_SCORE_M 2

/*
 * eti_score_prune_blocks -- the entropic keep set of half (b).
 *
 * For each sequence b, query head h and token i < ctx_lens[b]:
 *   x_i = scale * q[b,h,:] . k_i,   a_i = softmax_i(x_i) over all tokens,
 *   I_b^(h) = sum_{i in block} a_i I(v_i)
 * (Section 3.2; I(v_i) by score_mode, see above; tok_surp is read only in
 * mode E and must then be non-null), normalised to
 *   Ibar_b^(h) = n_b I_b^(h) / sum_b' I_b'^(h)   (1 when the sum is 0),
 * grouped per kv head as Ibar_b = max over the g query heads of the group.
 * Block b of (sequence, kv head) is kept iff Ibar_b >= theta[b_seq] (Section
 * 3.2) or b is among the first min(B_min, n_b) blocks ordered by (Ibar
 * descending, block index ascending) (minimum budget, Section 3.2).
 *
 * Outputs: keep_mask, kept_idx, kept_cnt (layouts above); block_score fp32
 * [B][Hkv][max_blocks] = Ibar (0 past n_b), nullable; token_scores and
 * kept_norm (layouts above), nullable together -- when given,
 * eti_paged_decode reuses them and reads no key page again.
 * theta: fp32 [B] (typically theta_next of the previous step; <= 0 keeps
 * every block, +inf keeps only the B_min budget).
 * A sequence with a bad page id or context length keeps nothing
 * (kept_cnt = 0) and gets its error bit.
 * Workspace: eti_score_prune_workspace_size(...) bytes.
 */
size_t eti_score_prune_workspace_size(int B, int Hq, int Hkv, int D, int P, int max_blocks);

int eti_score_prune_blocks(const eti_bf16* q, const eti_bf16* k_cache,
                           const int32_t* block_table, const int32_t* ctx_lens,
                           int B, int Hq, int Hkv, int D, int P, int max_blocks,
                           int64_t num_pages, float scale,
                           const float* theta, int B_min, int score_mode, const float* tok_surp,
                           uint8_t* keep_mask, int32_t* kept_idx, int32_t* kept_cnt,
                           float* block_score, float* token_scores, float* kept_norm,
                           uint32_t* err_flags, void* ws, size_t ws_bytes, void* stream);

/*
 * The two steps of eti_score_prune_blocks, callable separately (same
 * arguments and semantics; block_stats is the caller's buffer in place of the
 * workspace):
 *   eti_score_blocks  -- the scoring pass over every key page: token_scores
 *                        (nullable) and block_stats fp32 [B][Hkv][max_blocks][g][4]
 *                        = (m = max x, sum e^{x - m} - 1, sum e^{x - m}(x - m),
 *                        sum e^{x - m} s_i) per block and query head (the second
 *                        entry excludes one token at the max, which contributes
 *                        exactly 1, so it keeps full relative precision; the
 *                        fourth uses the stored surprisal s_i when tok_surp is
 *                        non-null and is 0 otherwise; garbage past n_b).
 *   eti_prune_blocks  -- the keep set, budget, compaction and kept-token
 *                        normaliser from block_stats in the given score_mode
 *                        (mode E needs stats made with tok_surp); writes
 *                        err_flags.
 * An unknown score_mode returns ETI_ERR_UNSUPPORTED.
 */
int eti_score_blocks(const eti_bf16* q, const eti_bf16* k_cache,
                     const int32_t* block_table, const int32_t* ctx_lens,
                     int B, int Hq, int Hkv, int D, int P, int max_blocks,
                     int64_t num_pages, float scale, const float* tok_surp,
                     float* token_scores, float* block_stats, void* stream);

int eti_prune_blocks(const float* block_stats, const int32_t* block_table,
                     const int32_t* ctx_lens, int B, int Hq, int Hkv, int D, int P,
                     int max_blocks, int64_t num_pages, const float* theta, int B_min,
                     int score_mode, uint8_t* keep_mask, int32_t* kept_idx, int32_t* kept_cnt,
                     float* block_score, float* kept_norm, uint32_t* err_flags, void* stream);

/*
 * eti_paged_decode -- GQA paged decode attention restricted to the kept
 * blocks (Section 3.2: attention computation is restricted to B_t; the
 * softmax is renormalised over the kept tokens):
 *   out[b,h,:] = sum_{i kept} softmax_kept(x_i) v_i,   x_i = scale q_h . k_i
 * out: bf16 [B][Hq][D].
 * The keep set comes from, in order of precedence: kept_idx + kept_cnt,
 * else keep_mask, else every block (dense decode).
 * When token_scores and kept_norm from eti_score_prune_blocks are given
 * (with kept_idx + kept_cnt from the same call), only the kept V pages and
 * kept scores are read; otherwise the keys of every block are scored first.
 * A sequence with no kept token, a bad page id or a bad context length gets
 * a zero output (and its error bit for the last two).
 * Workspace: eti_paged_decode_workspace_size(..., have_scores) bytes, where
 * have_scores says whether token_scores/kept_norm will be passed.
 */
size_t eti_paged_decode_workspace_size(int B, int Hq, int Hkv, int D, int P, int max_blocks,
                                       int have_scores);

int eti_paged_decode(const eti_bf16* q, const eti_bf16* k_cache, const eti_bf16* v_cache,
                     const int32_t* block_table, const int32_t* ctx_lens,
                     int B, int Hq, int Hkv, int D, int P, int max_blocks,
                     int64_t num_pages, float scale,
                     const uint8_t* keep_mask, const int32_t* kept_idx, const int32_t* kept_cnt,
                     const float* token_scores, const float* kept_norm,
                     eti_bf16* out, uint32_t* err_flags,
                     void* ws, size_t ws_bytes, void* stream);

/*
 * eti_set_wait_limit -- a diagnostic setting, not part of the method (the
 * paper has no counterpart): the number of polls after which a device-side
 * wait for a tile copy (in the scoring pass and in the decode pass) gives up
 * and reports ETI_ERRF_TIMEOUT for the sequences it serves.  It applies to
 * every call launched afterwards from this process, on every device; it is
 * the one setting of this library that outlives a call.  polls < 0 restores
 * the default (2^20 polls, far beyond any copy's latency).  0 makes every
 * such wait give up at once, which drives the error path without anything
 * being stuck: the copies already issued are still waited for, with the
 * default limit, before the kernel exits (ETI_ERRF_DRAIN if even that wait
 * gives up).  Returns the previous limit.
 */
int64_t eti_set_wait_limit(int64_t polls);

/* Version string and a readable name for a status code. */
const char* eti_version(void);
const char* eti_status_string(int status);

#ifdef __cplusplus
}
#endif

#endif /* ETI_H_ */
