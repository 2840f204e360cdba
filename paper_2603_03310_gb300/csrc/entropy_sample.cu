// entropy_sample.cu -- half (a) of the entropic-time decode step:
// entropy H_t of softmax(z / T_t) (Section 2.1), entropy flow and entropic
// time (Section 2), the temperature law (Section 3.3), the next pruning
// threshold (Section 3.2 safety floor, Section 5 entropy floor) and a
// Gumbel-max draw from p_t, in ONE pass over the fp32 logits and one launch
// (after a one-CTA kernel that zeroes the row tickets).
//
// Decomposition: a persistent grid of warps (24 per CTA, one CTA per SM) in
// which every warp takes an equal contiguous share of the row-major list of
// all rows' 4-token groups, so every SM finishes at the same time whatever B
// and V are.  There is no CTA-level barrier: a warp walks its share one row
// piece at a time, in steps of kG groups per lane (lane l takes groups
// base + 32 k + l, so its tokens are visited in increasing index order), with
// the next step's 16-byte loads in flight while the current one is
// processed.  Each lane keeps the online state
//     m  = running max of z (raw logit units),  mc = RD(m c), c = log2(e) / T
//          (the product rounded DOWN, so that t = z c - mc >= 0 exactly for
//          the tokens at the max and < 0 for the others, up to one ulp)
//     R  = sum of 2^t over the tokens below the max, t = fma(z, c, -mc)
//     N  = number of those tokens; nt = tokens seen - N are at the max, each of
//          weight 2^{t_max}, t_max = fma(m, c, -mc) in [0, ulp), so that
//          S = sum 2^t = nt 2^{t_max} + R
//     U  = sum 2^t * t
//     race best (r = w / E, index)  for the exponential race below.
// The rounding of mc shifts every t of a state by the same amount and cancels
// exactly in H = ln S - ln2 U / S.  Keeping the tokens at the max out of R (a
// 0/1 flag per token multiplies its weight) means a near-deterministic row
// (S = 1 + eps, eps down to 1e-6) keeps eps to full fp32 precision however
// many tokens a lane sums: no small weight is ever added to a value near 1.
// The per-token arithmetic runs on packed fp32 pairs (fma.rn.ftz.f32x2,
// add.rn.ftz.f32x2): two tokens per instruction for t, U, R, N and the race
// test; the tile max and the race test's minimum use 3-input max / min.
// At the end of a piece the warp reduces its lanes (max, rescale to it, then
// plain sums and the race argmax, in a fixed butterfly order), publishes the
// piece to slot (warp + row) and takes the row's ticket (an atomic, no
// waiting); the warp that takes the last ticket merges the row's slots in
// warp order (a fixed order: results do not depend on timing) and writes the
// per-row outputs.  A row that lies inside one warp's share is finalised
// from registers.
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
// shared by the warps of a CTA that work on the same row through a small
// table of one word per row in shared memory: a lane that reaches a new best
// publishes lr = log2 r + mc (the ratio in the row's common log2 frame) with
// a shared-memory atomicMax on the order-preserving key of lr, and every lane
// reads the word once per step and folds it into its own bound, 2^-10 shaved
// off for the rounding of lr and of its conversion back.  (One word per row in
// global memory, shared by the whole grid, was tried: the atomics on it cost
// more than the exact evaluations they saved.)  Before the first race of a
// piece every lane evaluates exactly the ratio of its own max token of the
// first step, and the warp publishes the best of them.  With
// fv = 1 + v - 2^-24, built from
// the word's bits with one logic op, the test is
//     fv - w / rk < 1 + 2^-21,
// one packed fma against -1/rk per token pair and a 3-input min over the
// step.  The 2^-21 slack covers the rounding of the fma and of 1/rk (for
// w / rk <= 1.6; every token with w / rk > 1 passes anyway), so no token with
// w > rk v is rejected; race_group then applies the per-token form
// fv < w / rk + 1 + 2^-21, which is conservative in the same way.
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

// 1 + v - 2^-24 from a word (v = 1 - u): the prefilter's left side.
__device__ __forceinline__ float fv_of(uint32_t word) {
    return __uint_as_float((~word & 0x7FFFFFu) | 0x3F800000u);
}

// ---- packed fp32 pairs (Blackwell f32x2 arithmetic, flush-to-zero) ----------
typedef unsigned long long f32x2;

__device__ __forceinline__ f32x2 pk2(float lo, float hi) {
    f32x2 r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}
__device__ __forceinline__ float2 up2(f32x2 v) {
    float2 r;
    asm("mov.b64 {%0, %1}, %2;" : "=f"(r.x), "=f"(r.y) : "l"(v));
    return r;
}
__device__ __forceinline__ f32x2 ffma2(f32x2 a, f32x2 b, f32x2 c) {
    f32x2 d;
    asm("fma.rn.ftz.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
    return d;
}
__device__ __forceinline__ f32x2 fadd2(f32x2 a, f32x2 b) {
    f32x2 d;
    asm("add.rn.ftz.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}
// max / min of three (a NaN operand is ignored, as for fmaxf / fminf)
__device__ __forceinline__ float max3f(float a, float b, float c) {
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}
__device__ __forceinline__ float min3f(float a, float b, float c) {
    float d;
    asm("min.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}
// 1.0 when t < 0, else 0.0 (NaN -> 0.0)
__device__ __forceinline__ float below0(float t) {
    float d;
    asm("set.lt.f32.f32 %0, %1, 0f00000000;" : "=f"(d) : "f"(t));
    return d;
}

// The frame of a state with max m: RD(m c).  Every kernel and merge forms it
// the same way, so states with equal maxima share it exactly.
__device__ __forceinline__ float frame_of(float m, float c) { return __fmul_rd(m, c); }

// Partial state of a row (piece), 24 bytes.  The frame mc = frame_of(m, c)
// is not stored.
//   m   max logit seen (raw units); -inf when empty
//   nt  number of tokens at m, each of weight 2^{t_max}, t_max = fma(m, c, -mc)
//   R   sum of 2^t over the other tokens (t = fma(z, c, -mc))
//   U   sum of 2^t t over all tokens
//   r   race best: w / E in this frame (0 = none);  bi: its token (INT_MAX = none)
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

// Merge partial `o` into `s` (both may be empty; c is the row's log2(e)/T):
// the state with the lower max is scaled into the other's frame, where all of
// its tokens are ordinary terms; equal maxima share the frame.
__device__ __forceinline__ void state_merge(RowState& s, RowState o, float c) {
    if (o.m == -kInf) {
        s.R += o.R;            // carries a NaN seen before any finite token
        return;
    }
    if (s.m == -kInf) { o.R += s.R; s = o; return; }
    if (o.m > s.m) { const RowState t = s; s = o; o = t; }
    float orr = o.r;
    if (o.m == s.m) {
        s.nt += o.nt;
        s.R += o.R;
        s.U += o.U;
    } else {
        const float smc = frame_of(s.m, c), omc = frame_of(o.m, c);
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

// Warp reduction of the lanes' states: the warp max, every lane rescaled to
// its frame, then butterfly sums and the race argmax (ties to the lower
// token).  Every lane ends with the same state; the order is fixed.
__device__ __forceinline__ void state_warp_reduce(RowState& s, float c) {
    float M = s.m;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
    if (s.m == -kInf) {
        s.nt = 0.f; s.U = 0.f; s.r = 0.f;
    } else if (s.m < M) {
        const float mc = frame_of(s.m, c), Mc = frame_of(M, c);
        const float d = mc - Mc;
        const float a = fast_ex2(d);
        const float S = state_sum(s, c, mc);
        s.U = a * fmaf(d, S, s.U);
        s.R = S * a;
        s.nt = 0.f;
        s.r *= a;
    }
    s.m = M;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        s.nt += __shfl_xor_sync(0xffffffffu, s.nt, o);
        s.R += __shfl_xor_sync(0xffffffffu, s.R, o);
        s.U += __shfl_xor_sync(0xffffffffu, s.U, o);
        const float orr = __shfl_xor_sync(0xffffffffu, s.r, o);
        const int obi = __shfl_xor_sync(0xffffffffu, s.bi, o);
        if (orr > s.r || (orr == s.r && obi < s.bi)) { s.r = orr; s.bi = obi; }
    }
}

// order-preserving int key of a float (and back); key(-inf) marks "no bound"
__device__ __forceinline__ int bound_key(float f) {
    const int b = __float_as_int(f);
    return b ^ ((b >> 31) & 0x7fffffff);
}
__device__ __forceinline__ float bound_unkey(int k) { return __int_as_float(k ^ ((k >> 31) & 0x7fffffff)); }
constexpr int kNoBound = (int)0x807fffff;   // bound_key(-inf)

constexpr float kRaceKappa = 1.4426950408889634f * (1.0f - 1.0f / 65536.0f);
constexpr float kPassC = 1.000000476837158203125f;    // 1 + 2^-21 >= (1 - 2^-24) + 2^-21 - rounding

// The exact race over one 4-token group (tokens x0 .. x0 + 3 in order, raw
// logits z) for the tokens that pass the per-token prefilter against
// 1/rk = ir.  The weights are recomputed exactly as the pass forms them.
// Kept out of line: it runs for a handful of groups per row piece.
struct RaceUpd {
    float r, rk;
    int bi, upd;
};
__device__ __noinline__ RaceUpd race_group(float4 z, uint4 wd4, float c, float mc, float ir, float r, int bi,
                                           float rk, int x0) {
    RaceUpd u{r, rk, bi, 0};
    const float zz[4] = {z.x, z.y, z.z, z.w};
    const uint32_t wd[4] = {wd4.x, wd4.y, wd4.z, wd4.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const float w = fast_ex2(fmaf(zz[e], c, -mc));
        if (fv_of(wd[e]) < fmaf(w, ir, kPassC)) {
            const float E = exp_variate_log2(wd[e]);
            if (w > u.r * E) {
                u.r = __fdividef(w, E);
                u.bi = x0 + e;
                u.rk = fmaxf(u.rk, fminf(u.r * kRaceKappa, 1e38f));
                ir = fast_rcp(u.rk);
                u.upd = 1;
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
    uint32_t off_lo, off_hi;
    unsigned long long* offset_dev;   // device offset (read at start; +1 by the last row), or null
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
    int nwarps;           // warps with a share
    int cta_warps;        // warps of a CTA that take shares (the others exit at once)
    long long share;      // groups per warp
    int* ticket;          // [B + 1]: pieces of each row published; [B]: rows finished
    RowState* part;       // [nwarps + B] partial states, slot (warp + row)
};

// 512 threads a CTA: alone as fast as 768, and beside the attention half of
// the step a little faster (the CTAs are placed in smaller pieces)
constexpr int kEtsThreads = 512;
constexpr int kEtsWarps = kEtsThreads / 32;
constexpr int kEtsCtasPerSm = 1;
constexpr int kBoundSlots = 32;        // rows of a CTA with a shared race bound
constexpr int kG = 2;                  // 4-token groups per lane per step
constexpr int kStep = 32 * kG;         // groups per warp step
constexpr int kMinGroupsPerWarp = 4 * kStep;   // below four steps a share is not worth a warp
constexpr float kFrameMax = 4096.f;    // |mc| above which lr loses the 2^-10 margin

constexpr int kRing = 4;               // warp steps in flight through the shared-memory ring
constexpr int kSlotBytes = kStep * 16; // one warp step of logits

// Direct loads of one step (rows off the 16-byte grid): the lane's kG groups
// as packed pairs, -inf outside [.., g1) and past V.
__device__ __forceinline__ void load_step_scalar(f32x2 (&z)[kG][2], const float* row, int gbase, int g1, int V) {
#pragma unroll
    for (int k = 0; k < kG; ++k) {
        const int g = gbase + 32 * k;
        float v[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int x = 4 * g + e;
            v[e] = (g < g1 && x < V) ? __ldg(row + x) : -kInf;
        }
        z[k][0] = pk2(v[0], v[1]);
        z[k][1] = pk2(v[2], v[3]);
    }
}

// Asynchronous copies of one step into a ring slot (16-byte aligned rows):
// lane l copies its groups gbase + 32 k to slot + k * 512 + 16 l.  A full
// group copies 16 bytes, the row's partial last group its valid bytes, a
// group outside [.., g1) nothing (the rest is zero-filled and masked later).
__device__ __forceinline__ void ring_issue(uint32_t slot, const float* row, int gbase, int g1, int V) {
#pragma unroll
    for (int k = 0; k < kG; ++k) {
        const int g = gbase + 32 * k;
        const int bytes = g < g1 ? min(16, max(0, (V - 4 * g) * 4)) : 0;
        const float* src = bytes > 0 ? row + 4 * (long long)g : row;
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;"
                     :: "r"(slot + (uint32_t)(k * 512)), "l"(src), "r"(bytes) : "memory");
    }
    cp_async_commit();
}

__device__ __forceinline__ void lds_2x2(f32x2& a, f32x2& b, uint32_t addr) {
    asm volatile("ld.shared.v2.b64 {%0, %1}, [%2];" : "=l"(a), "=l"(b) : "r"(addr) : "memory");
}

// The lane's pass over groups [g0, g1) of row b; returns its state.  With
// kVec the logits stream through the warp's ring of kRing step slots
// (cp.async, kRing - 1 steps ahead); otherwise one step is loaded ahead into
// registers.
template <bool kVec>
__device__ __forceinline__ RowState scan_piece(const EtsArgs& a, int b, int g0, int g1, float c,
                                               uint32_t off_lo, uint32_t off_hi, int lane, uint32_t ring,
                                               int* bound) {
    const float* row = a.logits + (long long)b * a.ld;
    const int full_groups = a.V >> 2;
    const int span = g1 - g0;
    const int nsteps = (span + kStep - 1) / kStep;
    const int g1f = min(g1, full_groups);
    const int nfast = g1f > g0 ? (g1f - g0) / kStep : 0;   // steps with every group full and inside
    float m = -kInf, mc = -kInf, nproc = 0.f;
    f32x2 R2 = pk2(0.f, 0.f), U2 = pk2(0.f, 0.f), N2 = pk2(0.f, 0.f);
    f32x2 c2 = pk2(c, c), nmc2 = pk2(0.f, 0.f), nir2 = pk2(-kInf, -kInf);
    float r = 0.f, rk = 0.f;
    int bi = 0x7fffffff;
    int seen = kNoBound, kb = kNoBound;
    const uint32_t lring = ring + 16 * lane;
    f32x2 cur[kG][2], nxt[kG][2];
    if (kVec) {
#pragma unroll
        for (int st = 0; st < kRing - 1; ++st) {
            if (st < nsteps) ring_issue(lring + st * kSlotBytes, row, g0 + st * kStep + lane, g1, a.V);
            else cp_async_commit();
        }
    } else {
        load_step_scalar(cur, row, g0 + lane, g1, a.V);
    }
#pragma unroll 1
    for (int it = 0; it < nsteps; ++it) {
        const int gb = g0 + it * kStep + lane;
        if (kVec) {
            const int ahead = it + kRing - 1;
            if (ahead < nsteps) ring_issue(lring + (ahead % kRing) * kSlotBytes, row, g0 + ahead * kStep + lane, g1, a.V);
            else cp_async_commit();
            cp_async_wait<kRing - 1>();           // this step's copies have landed
            const uint32_t sl = lring + (it % kRing) * kSlotBytes;
#pragma unroll
            for (int k = 0; k < kG; ++k) lds_2x2(cur[k][0], cur[k][1], sl + k * 512);
            if (it >= nfast) {
                // a ragged step: tokens outside [.., g1) or past V are -inf
#pragma unroll
                for (int k = 0; k < kG; ++k) {
                    const int g = gb + 32 * k;
                    float2 p = up2(cur[k][0]), q = up2(cur[k][1]);
                    const bool in = g < g1;
                    if (!(in && 4 * g < a.V)) p.x = -kInf;
                    if (!(in && 4 * g + 1 < a.V)) p.y = -kInf;
                    if (!(in && 4 * g + 2 < a.V)) q.x = -kInf;
                    if (!(in && 4 * g + 3 < a.V)) q.y = -kInf;
                    cur[k][0] = pk2(p.x, p.y);
                    cur[k][1] = pk2(q.x, q.y);
                }
            }
        } else if (it + 1 < nsteps) {
            load_step_scalar(nxt, row, gb + kStep, g1, a.V);
        }
        kb = *(volatile int*)bound;               // the bound the CTA's warps published
        // random words of this step's groups: the Philox chains do not depend
        // on the state, so they interleave with the loads in flight
        uint4 rr[kG];
#pragma unroll
        for (int k = 0; k < kG; ++k)
            rr[k] = philox4x32_10(make_uint4((uint32_t)(gb + 32 * k), (uint32_t)b, off_lo, off_hi), a.rk0, a.rk1);
        float bm = -kInf;
#pragma unroll
        for (int k = 0; k < kG; ++k) {
            const float2 p = up2(cur[k][0]), q = up2(cur[k][1]);
            bm = max3f(bm, p.x, p.y);
            bm = max3f(bm, q.x, q.y);
        }
        if (bm > m) {
            // a new max: the tokens at the old max become ordinary terms
            const float nmc = frame_of(bm, c);
            const float2 Rp = up2(R2), Up = up2(U2);
            float Rs = Rp.x + Rp.y, Us = Up.x + Up.y;
            if (m != -kInf) {
                const float2 Np = up2(N2);
                const float nt = nproc - (Np.x + Np.y);
                const float d = mc - nmc;                 // t_new = t_old + d
                const float sc = fast_ex2(d);
                const float S = fmaf(nt, fast_ex2(fmaf(m, c, -mc)), Rs);
                Us = sc * fmaf(d, S, Us);
                Rs = S * sc;
                r *= sc;
                rk *= sc;
            }
            R2 = pk2(Rs, 0.f);
            U2 = pk2(Us, 0.f);
            N2 = pk2(nproc, 0.f);
            m = bm;
            mc = nmc;
            nmc2 = pk2(-mc, -mc);
            const float nir = -fast_rcp(rk);
            nir2 = pk2(nir, nir);
        }
        if (it == 0) {
            // Seed the race bound before the first race: each lane evaluates
            // exactly the ratio of its max token of the step (a real token, so
            // a lower bound of the row's best); the warp keeps the largest.
            float lr = -kInf;
            if (m != -kInf && m < kInf && fabsf(mc) < kFrameMax) {
                uint32_t wd = 0;
                bool found = false;
#pragma unroll
                for (int k = 0; k < kG; ++k) {
                    const float2 p = up2(cur[k][0]), q = up2(cur[k][1]);
                    const float zz[4] = {p.x, p.y, q.x, q.y};
                    const uint32_t w4[4] = {rr[k].x, rr[k].y, rr[k].z, rr[k].w};
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        if (!found && zz[e] == m) { wd = w4[e]; found = true; }
                }
                const float r0 = __fdividef(fast_ex2(fmaf(m, c, -mc)), exp_variate_log2(wd));
                lr = fast_lg2(r0) + mc;
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) lr = fmaxf(lr, __shfl_xor_sync(0xffffffffu, lr, o));
            if (lane == 0 && lr != -kInf) atomicMax(bound, bound_key(lr));
            kb = max(kb, bound_key(lr));
        }
        if (kb != seen) {
            // a better bound was published for the row: fold it into ours
            seen = kb;
            if (m != -kInf && fabsf(mc) < kFrameMax) {
                const float rkb = fminf(fast_ex2(bound_unkey(kb) - mc - 0.0009765625f) * kRaceKappa, 1e38f);
                if (rkb > rk) {
                    rk = rkb;
                    const float nir = -fast_rcp(rk);
                    nir2 = pk2(nir, nir);
                }
            }
        }
        if (m == -kInf) {
            // no finite token yet: nothing to add or draw, but a NaN must
            // still poison the row
            bool nan = false;
#pragma unroll
            for (int k = 0; k < kG; ++k) {
                const float2 p = up2(cur[k][0]), q = up2(cur[k][1]);
                nan |= p.x != p.x || p.y != p.y || q.x != q.x || q.y != q.y;
            }
            if (nan) R2 = pk2(__int_as_float(0x7fc00000), 0.f);
        } else {
            float dmin = kInf;
#pragma unroll
            for (int k = 0; k < kG; ++k) {
                const uint32_t wd[4] = {rr[k].x, rr[k].y, rr[k].z, rr[k].w};
#pragma unroll
                for (int j = 0; j < 2; ++j) {
                    const f32x2 t2 = ffma2(cur[k][j], c2, nmc2);
                    const float2 t = up2(t2);
                    const float w0 = fast_ex2(t.x), w1 = fast_ex2(t.y);
                    const float tc0 = fmaxf(t.x, -250.f), tc1 = fmaxf(t.y, -250.f);   // -inf adds 0; NaN reaches U
                    const f32x2 w2 = pk2(w0, w1);
                    U2 = ffma2(w2, pk2(tc0, tc1), U2);
                    const f32x2 s2 = pk2(below0(tc0), below0(tc1));   // tokens at the max stay out of R
                    R2 = ffma2(w2, s2, R2);                           // (a NaN lands here)
                    N2 = fadd2(N2, s2);
                    const float2 d = up2(ffma2(w2, nir2, pk2(fv_of(wd[2 * j]), fv_of(wd[2 * j + 1]))));
                    dmin = min3f(dmin, d.x, d.y);
                }
            }
            if (dmin < kPassC) {
                // rare once the bound has formed: the exact race, in token order
#pragma unroll 1
                for (int k = 0; k < kG; ++k) {
                    const float2 p = up2(cur[k][0]), q = up2(cur[k][1]);
                    const RaceUpd u = race_group(make_float4(p.x, p.y, q.x, q.y), rr[k], c, mc,
                                                 -up2(nir2).x, r, bi, rk, 4 * (gb + 32 * k));
                    if (u.upd) {
                        r = u.r;
                        bi = u.bi;
                        rk = u.rk;
                        const float nir = -fast_rcp(rk);
                        nir2 = pk2(nir, nir);
                        if (fabsf(mc) < kFrameMax) atomicMax(bound, bound_key(fast_lg2(r) + mc));
                    }
                }
            }
        }
        nproc += 4.f * kG;
        if (!kVec) {
#pragma unroll
            for (int k = 0; k < kG; ++k) { cur[k][0] = nxt[k][0]; cur[k][1] = nxt[k][1]; }
        }
    }
    if (kVec) cp_async_wait<0>();   // (only empty groups can be left) before the ring is reused
    RowState s;
    const float2 Rp = up2(R2), Up = up2(U2), Np = up2(N2);
    s.m = m;
    s.R = Rp.x + Rp.y;
    s.U = m == -kInf ? 0.f : Up.x + Up.y;
    s.nt = m == -kInf ? 0.f : nproc - (Np.x + Np.y);
    s.r = r;
    s.bi = bi;
    return s;
}

// Outputs of row b from its merged state (one lane).
__device__ void row_epilogue(const EtsArgs& a, int b, const RowState& t, float c, bool bad_T) {
    const float Tt = a.T_in[b];
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
        // S = nt 2^{t_max} + R with 0 <= t_max < 2^-10, so 2^{t_max} = 1 + t_max ln2
        // to well below fp32 precision; ln S = ln nt + log1p(q), q = S / nt - 1
        const float mc = frame_of(t.m, c);
        const float q = fmaf(t.nt, fmaf(t.m, c, -mc) * kLn2, t.R) / t.nt;
        const float lnS = logf(t.nt) + log1pf(q);
        const float H = fmaxf(lnS - kLn2 * t.U / (t.nt * (1.f + q)), 0.f);
        const float H_prev = a.H_prev[b];
        const float dH = H_prev - H;
        a.tau[b] = a.tau[b] + fmaxf(dH, 0.f);
        float Tn = Tt * expf(a.p.sign * a.p.eta * (H - a.H_target[b]));
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
                const float tp = a.theta_next[b];   // the previous threshold, in place
                if (isfinite(tp)) th = fminf(tp + a.p.dtheta, fmaxf(tp - a.p.dtheta, th));
            }
            a.theta_next[b] = th;
        }
        if ((a.surprisal || a.surp_store) && t.bi >= 0 && t.bi < a.V) {
            const float tt = fmaf(a.logits[(long long)b * a.ld + t.bi], c, -mc);
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

// The pass: warp w takes groups [w*share, (w+1)*share) of the row-major list
// of all rows' 4-token groups, one row piece at a time.
template <bool kVec>
__global__ void __launch_bounds__(kEtsThreads, kEtsCtasPerSm)
entropy_sample_kernel(const __grid_constant__ EtsArgs a) {
    pdl_trigger();
    pdl_wait();
    extern __shared__ __align__(16) unsigned char ring_smem[];   // kVec: kEtsWarps * kRing * kSlotBytes
    // race bounds: one word for each of the first kBoundSlots rows of the CTA's
    // range, shared by its warps; a row beyond them uses a word of its warp's own
    __shared__ int bound_tab[kBoundSlots + kEtsWarps];
    const int lane = threadIdx.x & 31, wl = threadIdx.x >> 5;
    const int warp = blockIdx.x * a.cta_warps + wl;
    const uint32_t ring = smem_u32(ring_smem) + (uint32_t)(wl * kRing * kSlotBytes);
    for (int i = threadIdx.x; i < kBoundSlots + kEtsWarps; i += kEtsThreads) bound_tab[i] = kNoBound;
    const int row0 = (int)(min((long long)blockIdx.x * a.cta_warps * a.share, (long long)a.B * a.ngroups - 1) / a.ngroups);
    __syncthreads();
    if (wl >= a.cta_warps || warp >= a.nwarps) return;
    uint32_t off_lo = a.off_lo, off_hi = a.off_hi;
    if (a.offset_dev) {
        const unsigned long long o = *(volatile unsigned long long*)a.offset_dev;
        off_lo = (uint32_t)o;
        off_hi = (uint32_t)(o >> 32);
    }
    const long long total = (long long)a.B * a.ngroups;
    long long q0 = (long long)warp * a.share;
    const long long q1 = min(q0 + a.share, total);
    while (q0 < q1) {
        const int b = (int)(q0 / a.ngroups);
        const int g0 = (int)(q0 - (long long)b * a.ngroups);
        const int g1 = (int)min((long long)a.ngroups, q1 - (long long)b * a.ngroups);
        const float T = a.T_in[b] * a.p.T_cal;   // calibrated logits at temperature T_t
        const bool bad_T = !(T > 0.f && T < kInf);
        const float c = bad_T ? 0.f : kLog2e / T;
        RowState s;
        if (bad_T) state_init(s);
        else {
            int* bound = b - row0 < kBoundSlots ? bound_tab + (b - row0) : bound_tab + kBoundSlots + wl;
            if (b - row0 >= kBoundSlots) *(volatile int*)bound = kNoBound;   // the warp's own word, per row
            __syncwarp();
            s = scan_piece<kVec>(a, b, g0, g1, c, off_lo, off_hi, lane, ring, bound);
        }
        state_warp_reduce(s, c);
        const long long lo = (long long)b * a.ngroups, hi = lo + a.ngroups - 1;
        const int w0 = (int)(lo / a.share), w1 = (int)(hi / a.share);
        bool last = true;
        if (w1 > w0) {
            // publish the piece, then take the row's ticket (no waiting)
            int l = 0;
            if (lane == 0) {
                a.part[warp + b] = s;
                __threadfence();
                l = atomicAdd(a.ticket + b, 1) == w1 - w0;
            }
            last = __shfl_sync(0xffffffffu, l, 0) != 0;
            if (last) {
                __threadfence();
                // lane l merges slots w0 + l, w0 + l + 32, ... in order, then the
                // lanes merge in a fixed tree: the result does not depend on timing
                state_init(s);
                for (int w = w0 + lane; w <= w1; w += 32) {
                    const RowState* p = a.part + w + b;
                    RowState o;
                    o.m = __ldcg(&p->m); o.nt = __ldcg(&p->nt); o.R = __ldcg(&p->R);
                    o.U = __ldcg(&p->U); o.r = __ldcg(&p->r); o.bi = __ldcg(&p->bi);
                    state_merge(s, o, c);
                }
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    RowState o2 = state_shfl_xor(s, o);
                    if (lane & o) { const RowState t = o2; o2 = s; s = t; }   // lower lanes first
                    state_merge(s, o2, c);
                }
            }
        }
        if (last && lane == 0) {
            row_epilogue(a, b, s, c, bad_T);
            if (a.offset_dev) {
                // the last row to finish advances the device offset for the next call
                __threadfence();
                if (atomicAdd(a.ticket + a.B, 1) == a.B - 1) {
                    __threadfence();
                    *a.offset_dev = ((unsigned long long)off_hi << 32 | off_lo) + 1ull;
                }
            }
        }
        q0 = lo + g1;
    }
}

// Zeroes the row tickets (and the finished-row count) before the pass.
__global__ void __launch_bounds__(256) ets_clear_kernel(int* t, int n) {
    pdl_trigger();
    pdl_wait();
    for (int i = blockIdx.x * 256 + threadIdx.x; i < n; i += gridDim.x * 256) t[i] = 0;
}

}  // namespace eti

// Warps of the persistent sampling grid on the current device
static int ets_grid_warps() {
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    return eti::kEtsCtasPerSm * eti::kEtsWarps * sms;
}

static size_t ets_align256(size_t x) { return (x + 255) & ~size_t(255); }

// Scratch of one call: the tickets, then the partial states.
size_t eti_entropy_partial_bytes(int B) {
    return ets_align256((size_t)(B + 1) * sizeof(int)) + (size_t)(ets_grid_warps() + B) * sizeof(eti::RowState);
}

// Host launcher (called from the C ABI after argument validation); `scratch`
// holds eti_entropy_partial_bytes(B) bytes, 256-byte aligned.
int eti_launch_entropy_temp_sample(const float* logits, int B, int V, long long ld,
                                   const float* T_in, const float* H_prev, float* tau,
                                   const float* H_target, const eti_ctrl_params* p,
                                   uint64_t seed, uint64_t offset, uint64_t* offset_dev,
                                   int32_t* tok, float* H, float* T_out, float* dH,
                                   float* theta_next, float* surprisal,
                                   const eti_surp_store* store, uint32_t* err, void* scratch,
                                   cudaStream_t stream) {
    using namespace eti;
    if (B == 0) return ETI_OK;
    EtsArgs a;
    a.logits = logits; a.B = B; a.V = V; a.ld = ld; a.T_in = T_in; a.H_prev = H_prev;
    a.tau = tau; a.H_target = H_target; a.p = *p;
    const uint32_t seed_lo = (uint32_t)seed, seed_hi = (uint32_t)(seed >> 32);
    for (int r = 0; r < 10; ++r) {
        a.rk0[r] = seed_lo + (uint32_t)r * 0x9E3779B9u;
        a.rk1[r] = seed_hi + (uint32_t)r * 0xBB67AE85u;
    }
    a.off_lo = (uint32_t)offset; a.off_hi = (uint32_t)(offset >> 32);
    a.offset_dev = reinterpret_cast<unsigned long long*>(offset_dev);
    a.tok = tok; a.H = H; a.T_out = T_out; a.dH = dH; a.theta_next = theta_next;
    a.surprisal = surprisal; a.err = err;
    a.surp_store = store ? store->store : nullptr;
    a.slot_mapping = store ? store->slot_mapping : nullptr;
    a.num_slots = store ? (long long)store->num_slots : 0;
    a.ngroups = (V + 3) / 4;
    const long long total = (long long)B * a.ngroups;
    const int gw = ets_grid_warps();
    const long long want = (total + kMinGroupsPerWarp - 1) / kMinGroupsPerWarp;
    a.nwarps = (int)std::max(1LL, std::min((long long)gw, want));
    a.share = (total + a.nwarps - 1) / a.nwarps;
    // spread the warps over every SM: a small problem runs a few warps per CTA
    const int ctas = std::max(1, gw / kEtsWarps);
    a.cta_warps = std::min(kEtsWarps, (a.nwarps + ctas - 1) / ctas);
    char* sc = static_cast<char*>(scratch);
    a.ticket = reinterpret_cast<int*>(sc);
    a.part = reinterpret_cast<RowState*>(sc + ets_align256((size_t)(B + 1) * sizeof(int)));
    if (eti_launch_pdl(ets_clear_kernel, dim3((B + 1 + 255) / 256), dim3(256), 0, stream, a.ticket, B + 1) !=
        cudaSuccess)
        return ETI_ERR_CUDA;
    const bool vec = (ld % 4 == 0) && ((reinterpret_cast<uintptr_t>(logits) & 15) == 0);
    const dim3 grid((a.nwarps + a.cta_warps - 1) / a.cta_warps);
    cudaError_t e;
    if (vec) {
        const size_t smem = (size_t)kEtsWarps * kRing * kSlotBytes;
        if (cudaFuncSetAttribute(entropy_sample_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)smem) != cudaSuccess)
            return ETI_ERR_CUDA;
        e = eti_launch_pdl(entropy_sample_kernel<true>, grid, dim3(kEtsThreads), smem, stream, a);
    } else {
        e = eti_launch_pdl(entropy_sample_kernel<false>, grid, dim3(kEtsThreads), 0, stream, a);
    }
    return e == cudaSuccess ? ETI_OK : ETI_ERR_CUDA;
}

// ---------------------------------------------------------------------------
// eti_entropy_temp_sample_noalloc: the same computation with its scratch in a
// fixed array of this library instead of a caller workspace (see eti.h).

namespace {

constexpr size_t kNoAllocScratchBytes = 512 * 1024;
constexpr int kNoAllocMaxDevices = 64;

// One copy per device that loads the library; it lives until the process exits.
static __device__ __align__(256) unsigned char g_ets_scratch[kNoAllocScratchBytes];

// cuCtxGetCurrent, fetched from the driver at first use (no link dependency
// on libcuda): the cached address belongs to the context it was looked up in.
typedef CUresult (*CtxGetCurrentFn)(CUcontext*);

std::mutex g_ets_scratch_mu;
void* g_ets_scratch_ptr[kNoAllocMaxDevices] = {};
CUcontext g_ets_scratch_ctx[kNoAllocMaxDevices] = {};

// Device address of g_ets_scratch in the current context, looked up once per
// device and again whenever the device's current context changes (the
// host-side name of the array is not a device address).
int ets_scratch_address(void** out) {
    static CtxGetCurrentFn ctx_fn = nullptr;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return ETI_ERR_CUDA;
    if (dev < 0 || dev >= kNoAllocMaxDevices) return ETI_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_ets_scratch_mu);
    if (!ctx_fn) {
        void* fp = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &fp, 12000, cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess || !fp)
            return ETI_ERR_CUDA;
        ctx_fn = reinterpret_cast<CtxGetCurrentFn>(fp);
    }
    // make sure a context is current (the runtime creates the primary one)
    if (cudaFree(nullptr) != cudaSuccess) return ETI_ERR_CUDA;
    CUcontext ctx = nullptr;
    if (ctx_fn(&ctx) != CUDA_SUCCESS || !ctx) return ETI_ERR_CUDA;
    if (!g_ets_scratch_ptr[dev] || g_ets_scratch_ctx[dev] != ctx) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_ets_scratch) != cudaSuccess || !p) return ETI_ERR_CUDA;
        g_ets_scratch_ptr[dev] = p;
        g_ets_scratch_ctx[dev] = ctx;
    }
    *out = g_ets_scratch_ptr[dev];
    return ETI_OK;
}

}  // namespace

extern "C" size_t eti_entropy_temp_sample_noalloc_max_bytes(void) { return kNoAllocScratchBytes; }

extern "C" int eti_entropy_temp_sample_noalloc(const float* logits, int B, int V, int64_t ld,
                                               const float* T_in, const float* H_prev, float* tau,
                                               const float* H_target, const eti_ctrl_params* params,
                                               uint64_t seed, uint64_t offset, uint64_t* offset_dev,
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
                                          params, seed, offset, offset_dev, tok, H, T_out, dH,
                                          theta_next, tok_surprisal, surp_store, err_flags, scratch,
                                          (cudaStream_t)stream);
}
