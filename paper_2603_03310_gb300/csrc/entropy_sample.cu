// entropy_sample.cu -- half (a) of the entropic-time decode step:
// entropy H_t of softmax(z / T_t) (Section 2.1), entropy flow and entropic
// time (Section 2), the temperature law (Section 3.3), the next pruning
// threshold (Section 3.2 safety floor, Section 5 entropy floor) and a
// Gumbel-max draw from p_t, in ONE pass over the fp32 logits.
//
// Decomposition: a persistent grid (8 CTAs of 128 threads per SM) in which
// every CTA takes an equal contiguous share of the row-major list of all
// rows' 4-token groups, so every SM finishes at the same time whatever B and
// V are.  A CTA walks its share one row piece at a time, in steps of two
// groups per thread (thread t takes groups base + 128 k + t, so its tokens are
// visited in increasing index order), with the next step's 16-byte loads in
// flight while the current one is processed.  Each thread keeps the online
// state
//     m  = running max of z (raw logit units), mc = m * c,  c = log2(e) / T
//     nt = number of tokens equal to m,  R = sum of 2^{t} over the others,
//          t = z c - mc,  so that S = sum 2^{t} = nt 2^{t_max} + R
//     U  = sum 2^{t} * t
//     race best (r = w / E, index)  for the exponential race below.
// t is formed with one fma against the rounded mc; that rounding shifts every
// t of a state by the same amount and cancels exactly in H = ln S - ln2 U / S.
// Keeping the tokens at the max out of R (one compare and two selects per
// token) means a near-deterministic row (S = 1 + eps, eps down to 1e-6) keeps
// eps to full fp32 precision however many tokens a thread sums: no small
// weight is ever added to a value near 1.  A CTA writes one partial state per
// row piece it covered to scratch slot (cta + row); a finalize kernel merges
// each row's slots in CTA order (a fixed order: results do not depend on
// timing) and writes the per-row outputs.
//
// Sampling.  argmax_x y_x - log(-log u_x) is argmax_x w_x / E_x with
// w_x = exp(y_x - m) and the exponential variate E_x = -log u_x, so the
// exp() already needed for S is reused and one log per token remains.  The
// race keeps the best ratio r = w / E and a candidate wins when w > r E.
// E is computed in log2 units (the common factor cancels in the race):
//   u <= 15/16 : E2 = -lg2(u) with the MUFU approximation (|lg2 u| >= 0.093,
//                so its absolute error stays a small relative error);
//   u >  15/16 : v = 1 - u (exact), E2 = log2(e) * v * (1 + v/2 + ... + v^5/6),
//                the Taylor series of -log(1 - v), whose remainder is below
//                v^6/7 < 2^-24 / 7 relative.
// u = (2 (word & 0x7FFFFF) + 1) / 2^24 is formed exactly as 1.m - (1 - 2^-24).
//
// Race prefilter.  -log u >= 1 - u, so E2 >= log2(e) v with v = 1 - u, and
// both evaluations of E2 above stay within 2^-18 (relative) of the true
// value; a token with w <= rk v, rk = r_lb log2(e) (1 - 2^-16), therefore has
// w / E2 below r_lb by at least 2^-17 relative and cannot win, where r_lb is
// any ratio already reached in this row.  Only the tokens that pass evaluate
// E2 (out of line, in race_group), so the draw is unchanged.  The bound is
// shared by the whole CTA for its row piece: a thread that reaches a new best
// publishes lr = log2 r + mc (the ratio in the row's common frame) with a
// shared-memory atomicMax on the order-preserving key of lr, and every thread
// folds the published bound into its rk once per step, 2^-10 shaved off for
// the rounding of lr and of its conversion back.  Before the piece's first
// race every thread seeds the bound with the exact ratio of its own max token
// of the first step (one barrier), so that on the benchmark logits only a few
// dozen tokens per CTA piece reach the exact evaluation.  The test is
// evaluated as
//     1.f(~word) < w / rk + (1 - 2^-24) + 2^-21,
// the left side 1 + v - 2^-24 built from the word's bits with one logic op,
// the right side one fma against 1/rk.  The 2^-21 slack covers the rounding
// of the fma and of 1/rk (for w / rk <= 1.6; every token with w / rk > 1
// passes anyway), so no token that passes w > rk v is rejected; the slack
// also lets through the tokens with v within 2^-21 of w / rk.
#include <mutex>

#include "common.cuh"

namespace eti {

// Philox4x32-10 (Salmon et al., SC'11): ten rounds of two 32x32->64-bit
// multiplies; round r uses the key bumped r times by the Weyl constants.
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, const uint32_t (&k0)[10], const uint32_t (&k1)[10]) {
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        const unsigned long long p0 = (unsigned long long)0xD2511F53u * c.x;
        const unsigned long long p1 = (unsigned long long)0xCD9E8D57u * c.z;
        const uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
        const uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
        c = make_uint4(hi1 ^ c.y ^ k0[r], lo1, hi0 ^ c.w ^ k1[r], lo0);
    }
    return c;
}

// Exponential variate E / ln 2 from one 32-bit word (see the file comment).
__device__ __forceinline__ float exp_variate_log2(uint32_t word) {
    const float one_m = __uint_as_float((word & 0x7FFFFFu) | 0x3F800000u);   // 1 + j 2^-23
    const float u = one_m - __uint_as_float(0x3F7FFFFFu);                    // (2j + 1) 2^-24, exact
    const float v = 1.0f - u;                                                // exact for u > 1/2
    // log2(e) / (k + 1), k = 0..5
    float s = fmaf(v, 0.24044917348149393f, 0.28853900817779268f);
    s = fmaf(v, s, 0.36067376022224085f);
    s = fmaf(v, s, 0.48089834696298783f);
    s = fmaf(v, s, 0.72134752044448170f);
    s = fmaf(v, s, 1.4426950408889634f);
    const float series = v * s;
    const float direct = -fast_lg2(u);
    return u > 0.9375f ? series : direct;
}

// Partial state of a row (piece), 24 bytes.  The frame product mc = m c is
// not stored: it is recomputed from m and the row's c (always the same
// rounding) wherever it is needed.
//   m   max logit seen (raw units); -inf when empty
//   nt  number of tokens equal to m, each of weight 2^{t_max}, t_max = m c - mc
//   R   sum of 2^t over the other tokens (t = z c - mc)
//   U   sum of 2^t t over all tokens
//   r   race best: w / E in this frame (0 = none);  bi: its token (INT_MAX = none)
// Keeping the tokens at the max out of R means a near-deterministic row
// (S = 1 + eps, eps down to 1e-6) keeps eps to full fp32 precision: no small
// weight is ever added to a value near 1.
struct RowState {
    float m, nt, R, U, r;
    int bi;
};

__device__ __forceinline__ void state_init(RowState& s) {
    s.m = -kInf; s.nt = 0.f; s.R = 0.f; s.U = 0.f; s.r = 0.f; s.bi = 0x7fffffff;
}

// The state's S = sum 2^t in its own frame.
__device__ __forceinline__ float state_sum(const RowState& s, float c, float mc) {
    return fmaf(s.nt, fast_ex2(fmaf(s.m, c, -mc)), s.R);
}

// Move a thread's state to a new, larger max `nm` (its frame product in
// `mc`); the tokens at the old max become ordinary terms.  Returns the factor
// 2^{mc_old - mc_new} by which every earlier term was scaled.
__device__ __forceinline__ float state_rebase(RowState& s, float& mc, float nm, float c) {
    const float nmc = nm * c;
    float a = 0.f, d = 0.f, S = 0.f;
    if (s.m != -kInf) {
        d = mc - nmc;                            // t_new = t_old + d for every earlier term
        a = fast_ex2(d);
        S = state_sum(s, c, mc);
    }
    s.U = a * fmaf(d, S, s.U);
    s.R = S * a;
    s.nt = 0.f;
    s.r *= a;
    s.m = nm;
    mc = nmc;
    return a;
}

// Merge partial `o` into `s` (both may be empty; c is the row's log2(e)/T):
// the state with the lower max is scaled into the other's frame, where all of
// its tokens are ordinary terms; equal maxima share the frame.
__device__ __forceinline__ void state_merge(RowState& s, RowState o, float c) {
    if (o.m == -kInf) return;
    if (s.m == -kInf) { s = o; return; }
    if (o.m > s.m) { const RowState t = s; s = o; o = t; }
    float orr = o.r;
    if (o.m == s.m) {
        s.nt += o.nt;
        s.R += o.R;
        s.U += o.U;
    } else {
        const float smc = s.m * c, omc = o.m * c;
        const float d = omc - smc;               // < 0
        const float a = fast_ex2(d);
        const float So = state_sum(o, c, omc);
        s.U += a * fmaf(d, So, o.U);
        s.R = fmaf(So, a, s.R);
        orr *= a;
    }
    if (orr > s.r || (orr == s.r && o.bi < s.bi)) { s.r = orr; s.bi = o.bi; }
}

__device__ __forceinline__ RowState state_shfl_xor(const RowState& s, int o) {
    RowState r;
    r.m = __shfl_xor_sync(0xffffffffu, s.m, o);
    r.nt = __shfl_xor_sync(0xffffffffu, s.nt, o);
    r.R = __shfl_xor_sync(0xffffffffu, s.R, o);
    r.U = __shfl_xor_sync(0xffffffffu, s.U, o);
    r.r = __shfl_xor_sync(0xffffffffu, s.r, o);
    r.bi = __shfl_xor_sync(0xffffffffu, s.bi, o);
    return r;
}

constexpr float kRaceKappa = 1.4426950408889634f * (1.0f - 1.0f / 65536.0f);
constexpr float kPassC = 1.000000476837158203125f;    // 1 + 2^-21 >= (1 - 2^-24) + 2^-21 - rounding

// The exact race over one 4-token group (tokens x0 .. x0 + 3 in order) for the
// tokens that pass the prefilter against 1/rk = ir.  Kept out of line: it
// runs for a handful of groups per row piece, and inlined it would cost the
// straight path its registers and issue slots.
struct RaceUpd {
    float r, rk;
    int bi, pub;
};
__device__ __noinline__ RaceUpd race_group(float4 w4, uint4 wd4, float ir, float r, int bi, float rk, int x0) {
    RaceUpd u{r, rk, bi, 0};
    const float w[4] = {w4.x, w4.y, w4.z, w4.w};
    const uint32_t wd[4] = {wd4.x, wd4.y, wd4.z, wd4.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const float fv = __uint_as_float((~wd[e] & 0x7FFFFFu) | 0x3F800000u);
        if (fv < fmaf(w[e], ir, kPassC)) {
            const float E = exp_variate_log2(wd[e]);
            if (w[e] > u.r * E) {
                u.r = __fdividef(w[e], E);
                u.bi = x0 + e;
                u.rk = fmaxf(u.rk, fminf(u.r * kRaceKappa, 1e38f));
                ir = fast_rcp(u.rk);
                u.pub = 1;
            }
        }
    }
    return u;
}

struct EtsArgs {
    const float* logits;
    int B, V;
    long long ld;
    const float* T_in;
    const float* H_prev;
    float* tau;
    const float* H_target;
    eti_ctrl_params p;
    uint32_t seed_lo, seed_hi, off_lo, off_hi;
    uint32_t rk0[10], rk1[10];   // Philox round keys (the key bumped r times); the kernels
                                 // read them from the parameter bank, not from registers
    int32_t* tok;
    float* H;
    float* T_out;
    float* dH;
    float* theta_next;
    float* surprisal;
    float* surp_store;             // token-surprisal store (score mode E), or null
    const int64_t* slot_mapping;   // [B] slot of the drawn token in surp_store
    long long num_slots;
    uint32_t* err;
    int ngroups;          // 4-token groups per row
    long long share;      // groups per CTA of the grid
    RowState* part;       // [grid + B] partial states, slot (cta + row)
};

constexpr int kEtsThreads = 128;
constexpr int kEtsWarps = kEtsThreads / 32;
constexpr int kEtsPair = 2;        // 4-token groups per thread per step
constexpr int kEtsCtasPerSm = 8;
constexpr float kFrameMax = 4096.f;   // |mc| above which lr loses the 2^-10 margin

// order-preserving int key of a float (and back); key(-inf) marks "no bound"
__device__ __forceinline__ int bound_key(float f) {
    const int b = __float_as_int(f);
    return b ^ ((b >> 31) & 0x7fffffff);
}
__device__ __forceinline__ float bound_unkey(int k) { return __int_as_float(k ^ ((k >> 31) & 0x7fffffff)); }
constexpr int kNoBound = (int)0x807fffff;   // bound_key(-inf)

template <bool kVec>
__device__ __forceinline__ void load_group(float (&z)[4], const float* row, int g, int g1, int full_groups,
                                           int V) {
    if (kVec && g < g1 && g < full_groups) {
        const float4 v = ldg_stream_f4(row + 4 * (long long)g);
        z[0] = v.x; z[1] = v.y; z[2] = v.z; z[3] = v.w;
    } else {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int x = 4 * g + e;
            z[e] = (g < g1 && x < V) ? __ldg(row + x) : -kInf;
        }
    }
}

// The pass over the logits: CTA c takes groups [c*share, (c+1)*share) of the
// row-major list of all rows' 4-token groups, one row piece at a time; a
// piece is walked in steps of kEtsPair groups per thread (thread t takes
// groups base + k * 256 + t), the next step's 16-byte loads in flight while
// the current one is processed.
template <bool kVec>
__global__ void __launch_bounds__(kEtsThreads, kEtsCtasPerSm)
entropy_sample_partial_kernel(const __grid_constant__ EtsArgs a) {
    pdl_trigger();
    pdl_wait();
    __shared__ RowState warp_part[kEtsWarps];
    __shared__ int bound;   // the piece's race bound: key of the best lr, or kNoBound
    const int tid = threadIdx.x, lane = tid & 31;
    const long long total = (long long)a.B * a.ngroups;
    long long q0 = (long long)blockIdx.x * a.share;
    const long long q1 = min(q0 + a.share, total);
    const int full_groups = a.V >> 2;
    constexpr int step = kEtsPair * kEtsThreads;
    while (q0 < q1) {
        const int b = (int)(q0 / a.ngroups);
        const int g0 = (int)(q0 - (long long)b * a.ngroups);
        const int g1 = (int)min((long long)a.ngroups, q1 - (long long)b * a.ngroups);
        const float T = a.T_in[b] * a.p.T_cal;   // calibrated logits at temperature T_t
        const bool bad_T = !(T > 0.f && T < kInf);
        const float c = bad_T ? 0.f : kLog2e / T;
        const float* row = a.logits + (long long)b * a.ld;
        if (tid == 0) bound = kNoBound;
        __syncthreads();
        RowState s;
        state_init(s);
        float mc = -kInf, rk = 0.f, ir = kInf;
        int seen = kNoBound;
        if (!bad_T) {
            const int nsteps = (g1 - g0 + step - 1) / step;   // the same for every thread
            float cur[kEtsPair][4], nxt[kEtsPair][4];
#pragma unroll
            for (int k = 0; k < kEtsPair; ++k) load_group<kVec>(cur[k], row, g0 + k * kEtsThreads + tid, g1, full_groups, a.V);
            for (int it = 0; it < nsteps; ++it) {
                const int base = g0 + it * step;
                if (it + 1 < nsteps) {
#pragma unroll
                    for (int k = 0; k < kEtsPair; ++k)
                        load_group<kVec>(nxt[k], row, base + step + k * kEtsThreads + tid, g1, full_groups, a.V);
                }
                // random words of this step's groups, in one straight block so
                // that the Philox chains (independent of the state) interleave
                uint4 rr[kEtsPair];
#pragma unroll
                for (int k = 0; k < kEtsPair; ++k)
                    rr[k] = philox4x32_10(make_uint4((uint32_t)(base + k * kEtsThreads + tid), (uint32_t)b,
                                                     a.off_lo, a.off_hi), a.rk0, a.rk1);
                float bm = -kInf;
#pragma unroll
                for (int k = 0; k < kEtsPair; ++k)
#pragma unroll
                    for (int e = 0; e < 4; ++e) bm = fmaxf(bm, cur[k][e]);
                if (bm > s.m) {
                    rk *= state_rebase(s, mc, bm, c);
                    ir = fast_rcp(rk);
                }
                if (it == 0) {
                    // Seed the piece's race bound before its first race: each
                    // thread evaluates exactly the ratio of its max token of the
                    // step (a real token, so a lower bound of the row's best)
                    // and the CTA keeps the largest.
                    if (s.m != -kInf && s.m < kInf && fabsf(mc) < kFrameMax) {
                        uint32_t wd = 0;
                        bool found = false;
#pragma unroll
                        for (int k = 0; k < kEtsPair; ++k) {
                            const uint32_t w4[4] = {rr[k].x, rr[k].y, rr[k].z, rr[k].w};
#pragma unroll
                            for (int e = 0; e < 4; ++e)
                                if (!found && cur[k][e] == s.m) { wd = w4[e]; found = true; }
                        }
                        const float r0 = __fdividef(fast_ex2(fmaf(s.m, c, -mc)), exp_variate_log2(wd));
                        atomicMax(&bound, bound_key(fast_lg2(r0) + mc));
                    }
                    __syncthreads();
                }
                if (s.m == -kInf) {
                    // no finite token yet: nothing to add or draw, but a NaN
                    // must still poison the row
                    bool nan = false;
#pragma unroll
                    for (int k = 0; k < kEtsPair; ++k)
#pragma unroll
                        for (int e = 0; e < 4; ++e) nan |= cur[k][e] != cur[k][e];
                    if (nan) s.R = __int_as_float(0x7fc00000);
                } else {
                    const int kb = *(volatile int*)&bound;
                    if (kb != seen) {
                        seen = kb;
                        if (fabsf(mc) < kFrameMax) {
                            const float rkb = fminf(fast_ex2(bound_unkey(kb) - mc - 0.0009765625f) * kRaceKappa, 1e38f);
                            if (rkb > rk) {
                                rk = rkb;
                                ir = fast_rcp(rk);
                            }
                        }
                    }
#pragma unroll
                    for (int k = 0; k < kEtsPair; ++k) {
                        float w[4];
                        const uint32_t wd[4] = {rr[k].x, rr[k].y, rr[k].z, rr[k].w};
                        bool any = false;
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const float t = fmaf(cur[k][e], c, -mc);
                            w[e] = fast_ex2(t);
                            s.U = fmaf(w[e], fmaxf(t, -250.f), s.U);   // -inf adds 0; NaN reaches U
                            const bool at_max = cur[k][e] == s.m;      // the tokens at the max stay out of R
                            s.nt += at_max ? 1.f : 0.f;
                            s.R += at_max ? 0.f : w[e];                 // (a NaN lands here)
                            const float fv = __uint_as_float((~wd[e] & 0x7FFFFFu) | 0x3F800000u);
                            any |= fv < fmaf(w[e], ir, kPassC);
                        }
                        if (any) {
                            // rare once the bound has formed: the exact race, in token order
                            const RaceUpd u = race_group(make_float4(w[0], w[1], w[2], w[3]), rr[k], ir, s.r, s.bi,
                                                         rk, 4 * (base + k * kEtsThreads + tid));
                            if (u.pub) {
                                s.r = u.r;
                                s.bi = u.bi;
                                rk = u.rk;
                                ir = fast_rcp(rk);
                                if (fabsf(mc) < kFrameMax) atomicMax(&bound, bound_key(fast_lg2(s.r) + mc));
                            }
                        }
                    }
                }
#pragma unroll
                for (int k = 0; k < kEtsPair; ++k)
#pragma unroll
                    for (int e = 0; e < 4; ++e) cur[k][e] = nxt[k][e];
            }
        }
        // CTA reduction of the piece into slot (cta + row), in a fixed order
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) state_merge(s, state_shfl_xor(s, o), c);
        if (lane == 0) warp_part[tid >> 5] = s;
        __syncthreads();
        if (tid == 0) {
            RowState t = warp_part[0];
            for (int w = 1; w < kEtsWarps; ++w) state_merge(t, warp_part[w], c);
            a.part[blockIdx.x + b] = t;
        }
        q0 = (long long)b * a.ngroups + g1;
    }
}

// Per row: merge the partial slots in CTA order, then the scalar epilogue.
__global__ void __launch_bounds__(128)
entropy_sample_finalize_kernel(const EtsArgs a) {
    pdl_trigger();
    pdl_wait();
    const int lane = threadIdx.x & 31;
    const int b = blockIdx.x * 4 + (threadIdx.x >> 5);
    if (b >= a.B) return;
    const float Tt = a.T_in[b];
    const float T = Tt * a.p.T_cal;              // calibrated logits at temperature T_t
    const bool bad_T = !(T > 0.f && T < kInf);
    const float c = bad_T ? 0.f : kLog2e / T;
    const long long lo = (long long)b * a.ngroups, hi = lo + a.ngroups - 1;
    const int c0 = (int)(lo / a.share), c1 = (int)(hi / a.share);
    // the per-row inputs of the epilogue, loaded while the slots are merged
    float tau_in = 0.f, H_prev = 0.f, H_tgt = 0.f, th_prev = 0.f;
    if (lane == 0) {
        tau_in = a.tau[b];
        H_prev = a.H_prev[b];
        H_tgt = a.H_target[b];
        if (a.theta_next && a.p.dtheta > 0.f) th_prev = a.theta_next[b];
    }
    // lane l merges slots c0 + l, c0 + l + 32, ... in order, then the lanes merge
    // in a fixed tree: the result does not depend on timing
    RowState s;
    state_init(s);
    for (int cc = c0 + lane; cc <= c1; cc += 32) state_merge(s, a.part[cc + b], c);
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        RowState o2 = state_shfl_xor(s, o);
        // keep the lower-lane state first (a fixed order of the sums)
        if (lane & o) { RowState t = o2; o2 = s; s = t; }
        state_merge(s, o2, c);
    }
    if (lane != 0) return;
    const RowState& t = s;
    const float* row = a.logits + (long long)b * a.ld;
    uint32_t err = bad_T ? ETI_ERRF_BAD_TEMP : 0u;
    if (!err) {
        if (t.m == -kInf) err = ETI_ERRF_ALL_NEG_INF;
        else if (t.m == kInf || isnan(t.R) || isnan(t.U)) err = ETI_ERRF_NONFINITE;
    }
    if (err) {
        a.tok[b] = -1;
        a.H[b] = __int_as_float(0x7fc00000);
        a.T_out[b] = Tt;
        if (a.dH) a.dH[b] = __int_as_float(0x7fc00000);
        if (a.theta_next) a.theta_next[b] = 0.f;
        if (a.surprisal) a.surprisal[b] = __int_as_float(0x7fc00000);
    } else {
        // S = nt 2^{t_max} + R with |t_max| < 2^-10, so 2^{t_max} = 1 + t_max ln2
        // to well below fp32 precision; ln S = ln nt + log1p(q), q = S / nt - 1
        const float mc = t.m * c;
        const float q = fmaf(t.nt, fmaf(t.m, c, -mc) * kLn2, t.R) / t.nt;
        const float lnS = logf(t.nt) + log1pf(q);
        const float H = fmaxf(lnS - kLn2 * t.U / (t.nt * (1.f + q)), 0.f);
        const float dH = H_prev - H;
        a.tau[b] = tau_in + fmaxf(dH, 0.f);
        float Tn = Tt * expf(a.p.sign * a.p.eta * (H - H_tgt));
        if (a.p.rho_T > 0.f) Tn = fminf(Tt * expf(a.p.rho_T), fmaxf(Tt * expf(-a.p.rho_T), Tn));
        Tn = fminf(a.p.T_max, fmaxf(a.p.T_min, Tn));
        a.tok[b] = t.bi;
        a.H[b] = H;
        a.T_out[b] = Tn;
        if (a.dH) a.dH[b] = dH;
        if (a.theta_next) {
            const float Heff = fmaxf(H - a.p.eps_H, a.p.H_min);
            const float tmax = a.V > 1 ? a.p.theta_hi * fmaxf(0.f, 1.f - Heff / logf((float)a.V))
                                       : a.p.theta_hi;
            float th = fminf(a.p.theta_user, tmax);
            if (a.p.dtheta > 0.f) {
                const float tp = th_prev;   // the previous threshold, in place
                if (isfinite(tp)) th = fminf(tp + a.p.dtheta, fmaxf(tp - a.p.dtheta, th));
            }
            a.theta_next[b] = th;
        }
        if (a.surprisal || a.surp_store) {
            const float tt = fmaf(row[t.bi], c, -mc);
            const float sp = lnS - kLn2 * tt;
            if (a.surprisal) a.surprisal[b] = sp;
            if (a.surp_store) {
                const long long slot = a.slot_mapping[b];
                if (slot >= 0 && slot < a.num_slots) a.surp_store[slot] = sp;
            }
        }
    }
    a.err[b] = err;
}

}  // namespace eti

// CTAs of the persistent sampling grid on the current device
int eti_entropy_ncta() {
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    return eti::kEtsCtasPerSm * sms;
}

size_t eti_entropy_partial_bytes(int B) {
    return (size_t)(eti_entropy_ncta() + B) * sizeof(eti::RowState);
}

// Host launcher (called from the C ABI after argument validation); `part`
// holds eti_entropy_partial_bytes(B) bytes of scratch.
int eti_launch_entropy_temp_sample(const float* logits, int B, int V, long long ld,
                                   const float* T_in, const float* H_prev, float* tau,
                                   const float* H_target, const eti_ctrl_params* p,
                                   uint64_t seed, uint64_t offset, int32_t* tok, float* H,
                                   float* T_out, float* dH, float* theta_next, float* surprisal,
                                   const eti_surp_store* store, uint32_t* err, void* part,
                                   cudaStream_t stream) {
    using namespace eti;
    if (B == 0) return ETI_OK;
    const int ncta = eti_entropy_ncta();
    EtsArgs a;
    a.logits = logits; a.B = B; a.V = V; a.ld = ld; a.T_in = T_in; a.H_prev = H_prev;
    a.tau = tau; a.H_target = H_target; a.p = *p;
    a.seed_lo = (uint32_t)seed; a.seed_hi = (uint32_t)(seed >> 32);
    for (int r = 0; r < 10; ++r) {
        a.rk0[r] = a.seed_lo + (uint32_t)r * 0x9E3779B9u;
        a.rk1[r] = a.seed_hi + (uint32_t)r * 0xBB67AE85u;
    }
    a.off_lo = (uint32_t)offset; a.off_hi = (uint32_t)(offset >> 32);
    a.tok = tok; a.H = H; a.T_out = T_out; a.dH = dH; a.theta_next = theta_next;
    a.surprisal = surprisal; a.err = err;
    a.surp_store = store ? store->store : nullptr;
    a.slot_mapping = store ? store->slot_mapping : nullptr;
    a.num_slots = store ? (long long)store->num_slots : 0;
    a.ngroups = (V + 3) / 4;
    const long long total = (long long)B * a.ngroups;
    a.part = static_cast<RowState*>(part);
    a.share = (total + ncta - 1) / ncta;
    const bool vec = (ld % 4 == 0) && ((reinterpret_cast<uintptr_t>(logits) & 15) == 0);
    const cudaError_t e1 = vec ? eti_launch_pdl(entropy_sample_partial_kernel<true>, dim3(ncta), dim3(kEtsThreads), 0, stream, a)
                               : eti_launch_pdl(entropy_sample_partial_kernel<false>, dim3(ncta), dim3(kEtsThreads), 0, stream, a);
    if (e1 != cudaSuccess) return ETI_ERR_CUDA;
    return eti_launch_pdl(entropy_sample_finalize_kernel, dim3((B + 3) / 4), dim3(128), 0, stream, a) == cudaSuccess
               ? ETI_OK : ETI_ERR_CUDA;
}

// ---------------------------------------------------------------------------
// eti_entropy_temp_sample_noalloc: the same computation with its scratch in a
// fixed array of this library instead of a caller workspace (see eti.h).

namespace {

constexpr size_t kNoAllocScratchBytes = 256 * 1024;
constexpr int kNoAllocMaxDevices = 64;

// One copy per device that loads the library; it lives until the process exits.
static __device__ __align__(256) unsigned char g_ets_scratch[kNoAllocScratchBytes];

std::mutex g_ets_scratch_mu;
void* g_ets_scratch_ptr[kNoAllocMaxDevices] = {};

// Device address of g_ets_scratch on the current device, looked up once per
// device (the host-side name of the array is not a device address).
int ets_scratch_address(void** out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return ETI_ERR_CUDA;
    if (dev < 0 || dev >= kNoAllocMaxDevices) return ETI_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_ets_scratch_mu);
    if (!g_ets_scratch_ptr[dev]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_ets_scratch) != cudaSuccess || !p) return ETI_ERR_CUDA;
        g_ets_scratch_ptr[dev] = p;
    }
    *out = g_ets_scratch_ptr[dev];
    return ETI_OK;
}

}  // namespace

extern "C" size_t eti_entropy_temp_sample_noalloc_max_bytes(void) { return kNoAllocScratchBytes; }

extern "C" int eti_entropy_temp_sample_noalloc(const float* logits, int B, int V, int64_t ld,
                                               const float* T_in, const float* H_prev, float* tau,
                                               const float* H_target, const eti_ctrl_params* params,
                                               uint64_t seed, uint64_t offset,
                                               int32_t* tok, float* H, float* T_out,
                                               float* dH, float* theta_next, float* tok_surprisal,
                                               const eti_surp_store* surp_store,
                                               uint32_t* err_flags, void* stream) {
    if (B < 0 || B > 65535 || V < 1 || ld < V) return ETI_ERR_SHAPE;
    if (B == 0) return ETI_OK;
    if (!logits || !T_in || !H_prev || !tau || !H_target || !params || !tok || !H || !T_out ||
        !err_flags)
        return ETI_ERR_NULL;
    if (surp_store && (!surp_store->store || !surp_store->slot_mapping)) return ETI_ERR_NULL;
    if (eti_entropy_partial_bytes(B) > kNoAllocScratchBytes) return ETI_ERR_TOO_LARGE;
    void* scratch = nullptr;
    const int st = ets_scratch_address(&scratch);
    if (st != ETI_OK) return st;
    return eti_launch_entropy_temp_sample(logits, B, V, (long long)ld, T_in, H_prev, tau, H_target,
                                          params, seed, offset, tok, H, T_out, dH, theta_next,
                                          tok_surprisal, surp_store, err_flags, scratch,
                                          (cudaStream_t)stream);
}
