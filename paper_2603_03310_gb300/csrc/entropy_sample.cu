// entropy_sample.cu -- half (a) of the entropic-time decode step:
// entropy H_t of softmax(z / T_t) (Section 2.1), entropy flow and entropic
// time (Section 2), the temperature law (Section 3.3), the next pruning
// threshold (Section 3.2 safety floor, Section 5 entropy floor) and a
// Gumbel-max draw from p_t, in ONE pass over the fp32 logits.
//
// Decomposition: a persistent grid (4 CTAs per SM) in which every CTA takes an
// equal contiguous share of the row-major list of all rows' 4-token groups,
// so every SM finishes at the same time whatever B and V are.  Each CTA
// streams its share with 128-bit loads (the next pair of groups is in flight
// while the current pair is processed) and keeps, per thread, the online state
//     m  = running max of z (raw logit units), mc = m * c,  c = log2(e) / T
//     S  = sum 2^{t},  t = z c - mc
//     U  = sum 2^{t} * t
//     race best (r = w / E, index)  for the exponential race below.
// t is formed with one fma against the rounded mc; that rounding shifts every
// t of a state by the same amount and cancels exactly in H = ln2 (log2 S - U/S).
// A CTA writes one partial state per row piece it covered to scratch slot
// (cta + row); a finalize kernel merges each row's slots in CTA order (a fixed
// order: results do not depend on timing) and writes the per-row outputs.
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

struct RowState {
    float m;    // max logit seen (raw units)
    float mc;   // m * c, rounded once
    float S;    // sum 2^t
    float U;    // sum 2^t * t
    float r;    // race best: w / E relative to m (0 = none)
    int bi;     // race best: token index (INT_MAX = none)
};

__device__ __forceinline__ void state_init(RowState& s) {
    s.m = -kInf; s.mc = -kInf; s.S = 0.f; s.U = 0.f; s.r = 0.f; s.bi = 0x7fffffff;
}

// Move the state to a new, larger reference max `nm`; returns the factor
// 2^{mc_old - mc_new} by which every term of the state was scaled.
__device__ __forceinline__ float state_rebase(RowState& s, float nm, float c) {
    const float nmc = nm * c;
    float a = 0.f, d = 0.f;
    if (s.m != -kInf) {
        d = s.mc - nmc;              // t_new = t_old + d for every term of the state
        a = fast_ex2(d);
    }
    s.U = a * fmaf(d, s.S, s.U);
    s.S *= a;
    s.r *= a;
    s.m = nm;
    s.mc = nmc;
    return a;
}

// Merge partial `o` into `s` (both may be empty).
__device__ __forceinline__ void state_merge(RowState& s, RowState o, float c) {
    if (o.m == -kInf) return;
    if (s.m == -kInf) { s = o; return; }
    if (o.m > s.m) {
        state_rebase(s, o.m, c);
        // align o to the same rounded reference
        const float d = o.mc - s.mc;
        const float a = fast_ex2(d);
        o.U = a * fmaf(d, o.S, o.U); o.S *= a; o.r *= a;
    } else {
        const float d = o.mc - s.mc;
        const float a = fast_ex2(d);
        o.U = a * fmaf(d, o.S, o.U); o.S *= a; o.r *= a;
    }
    s.S += o.S;
    s.U += o.U;
    if (o.r > s.r || (o.r == s.r && o.bi < s.bi)) { s.r = o.r; s.bi = o.bi; }
}

__device__ __forceinline__ RowState state_shfl_xor(const RowState& s, int o) {
    RowState r;
    r.m = __shfl_xor_sync(0xffffffffu, s.m, o);
    r.mc = __shfl_xor_sync(0xffffffffu, s.mc, o);
    r.S = __shfl_xor_sync(0xffffffffu, s.S, o);
    r.U = __shfl_xor_sync(0xffffffffu, s.U, o);
    r.r = __shfl_xor_sync(0xffffffffu, s.r, o);
    r.bi = __shfl_xor_sync(0xffffffffu, s.bi, o);
    return r;
}

// Race prefilter.  -log u >= 1 - u, so E2 >= log2(e) v with v = 1 - u, and
// both evaluations of E2 above stay within 2^-18 (relative) of the true
// value; a token with w <= rk v, rk = r_lb log2(e) (1 - 2^-16), therefore has
// w / E2 below r_lb by at least 2^-17 relative and cannot win, where r_lb is
// any ratio already reached in this row (own best, or a bound shared by the
// warp).  Only the tokens that pass evaluate E2, so the draw is unchanged.
constexpr float kRaceKappa = 1.4426950408889634f * (1.0f - 1.0f / 65536.0f);

// v = 1 - u = (2 (0x7FFFFF - j) + 1) 2^-24 for the word's uniform u, formed exactly
__device__ __forceinline__ float one_minus_u(uint32_t word) {
    return __uint_as_float((~word & 0x7FFFFFu) | 0x3F800000u) - __uint_as_float(0x3F7FFFFFu);
}

constexpr int kEtsThreads = 256;
constexpr int kEtsPair = 2;     // 4-token groups per thread per pipeline step
constexpr int kEtsCtasPerSm = 4;

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
    long long share;      // groups per CTA of the persistent grid
    RowState* part;       // [nCTA + B] partial states, slot (cta + row)
};

template <bool kVec>
__device__ __forceinline__ void load_group(float (&z)[4], const float* row, int g, int g1, int full_groups,
                                           int V) {
    if (g < g1 && kVec && g < full_groups) {
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

// Persistent pass: CTA c takes groups [c*share, (c+1)*share) of the
// row-major list of all rows' 4-token groups, one row piece at a time.
template <bool kVec>
__global__ void __launch_bounds__(kEtsThreads, kEtsCtasPerSm)
entropy_sample_partial_kernel(const __grid_constant__ EtsArgs a) {
    pdl_trigger();
    pdl_wait();
    __shared__ RowState warp_part[kEtsThreads / 32];
    const int tid = threadIdx.x;
    const long long total = (long long)a.B * a.ngroups;
    long long q0 = (long long)blockIdx.x * a.share;
    const long long q1 = min(q0 + a.share, total);
    const int full_groups = a.V >> 2;
    while (q0 < q1) {
        const int b = (int)(q0 / a.ngroups);
        const int g0 = (int)(q0 - (long long)b * a.ngroups);
        const int g1 = (int)min((long long)a.ngroups, q1 - (long long)b * a.ngroups);
        const float T = a.T_in[b] * a.p.T_cal;   // calibrated logits at temperature T_t
        const bool bad_T = !(T > 0.f && T < kInf);
        const float c = bad_T ? 0.f : kLog2e / T;
        const float* row = a.logits + (long long)b * a.ld;
        RowState s;
        state_init(s);
        float rk = 0.f;              // race prefilter bound, in the state's frame
        bool shared = false;         // the warp's bound has been folded into rk
        // every lane of the warp walks this row piece (the same steps), so the
        // warp may exchange its bound with full-mask shuffles
        const bool warp_full = g0 + (tid | 31) < g1;
        if (!bad_T && g0 + tid < g1) {
            constexpr int step = kEtsPair * kEtsThreads;
            float cur[kEtsPair][4], nxt[kEtsPair][4];
#pragma unroll
            for (int k = 0; k < kEtsPair; ++k) load_group<kVec>(cur[k], row, g0 + k * kEtsThreads + tid, g1, full_groups, a.V);
            for (int base = g0; base < g1; base += step) {
                const bool more = base + step < g1;
                if (more) {
#pragma unroll
                    for (int k = 0; k < kEtsPair; ++k)
                        load_group<kVec>(nxt[k], row, base + step + k * kEtsThreads + tid, g1, full_groups, a.V);
                }
                float bm = -kInf;
#pragma unroll
                for (int k = 0; k < kEtsPair; ++k)
#pragma unroll
                    for (int e = 0; e < 4; ++e) bm = fmaxf(bm, cur[k][e]);
                if (bm == -kInf) {
                    // every token of the pair is -inf (or NaN): nothing to add and
                    // nothing to draw, but a NaN must still poison the row
                    bool nan = false;
#pragma unroll
                    for (int k = 0; k < kEtsPair; ++k)
#pragma unroll
                        for (int e = 0; e < 4; ++e) nan |= (cur[k][e] != cur[k][e]);
                    if (nan) s.S = __int_as_float(0x7fc00000);
                } else {
                    if (bm > s.m) rk *= state_rebase(s, bm, c);
                    // entropy sums for every token, the race prefilter folded into
                    // one flag; groups past the piece hold -inf (w = 0, never drawn)
                    float w[kEtsPair][4];
                    uint32_t word[kEtsPair][4];
                    bool any = false;
#pragma unroll
                    for (int k = 0; k < kEtsPair; ++k) {
                        const int g = base + k * kEtsThreads + tid;
                        const uint4 r = philox4x32_10(make_uint4((uint32_t)g, (uint32_t)b, a.off_lo, a.off_hi), a.rk0, a.rk1);
                        word[k][0] = r.x; word[k][1] = r.y; word[k][2] = r.z; word[k][3] = r.w;
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const float t = fmaf(cur[k][e], c, -s.mc);
                            w[k][e] = fast_ex2(t);
                            s.S += w[k][e];
                            s.U = fmaf(w[k][e], fmaxf(t, -250.f), s.U);   // -inf adds 0; NaN reaches S
                            any |= w[k][e] > rk * one_minus_u(word[k][e]);
                        }
                    }
                    if (any) {
                        // rare once rk has grown: the exact race, in token order
#pragma unroll
                        for (int k = 0; k < kEtsPair; ++k)
#pragma unroll
                            for (int e = 0; e < 4; ++e)
                                if (w[k][e] > rk * one_minus_u(word[k][e])) {
                                    const float E = exp_variate_log2(word[k][e]);
                                    if (w[k][e] > s.r * E) {
                                        s.r = __fdividef(w[k][e], E);
                                        s.bi = 4 * (base + k * kEtsThreads + tid) + e;
                                        rk = fmaxf(rk, s.r * kRaceKappa);
                                    }
                                }
                    }
                }
                if (!more) break;
                if (!shared && warp_full) {
                    // After the first step, share the best ratio of the warp as
                    // a bound: lr = log2 r + mc is the ratio in the row's common
                    // frame, and the 2^-10 shaved off covers the rounding of
                    // lr and of its conversion back to this state's frame.  The
                    // cap keeps rk finite, so a later rebase by 0 gives 0.
                    shared = true;
                    float lr = s.r > 0.f ? fast_lg2(s.r) + s.mc : -kInf;
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1) lr = fmaxf(lr, __shfl_xor_sync(0xffffffffu, lr, o));
                    if (lr > -kInf && s.m != -kInf)
                        rk = fmaxf(rk, fminf(fast_ex2(lr - s.mc - 0.0009765625f) * kRaceKappa, 1e38f));
                }
#pragma unroll
                for (int k = 0; k < kEtsPair; ++k)
#pragma unroll
                    for (int e = 0; e < 4; ++e) cur[k][e] = nxt[k][e];
            }
        }
        // CTA reduction of the piece into slot (cta + row)
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) state_merge(s, state_shfl_xor(s, o), c);
        if ((tid & 31) == 0) warp_part[tid >> 5] = s;
        __syncthreads();
        if (tid == 0) {
            RowState t = warp_part[0];
            for (int w = 1; w < kEtsThreads / 32; ++w) state_merge(t, warp_part[w], c);
            a.part[blockIdx.x + b] = t;
        }
        __syncthreads();
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
    // lane l merges slots c0 + l, c0 + l + 32, ... in order, then the lanes merge
    // in a fixed tree: the result does not depend on timing
    RowState s;
    state_init(s);
    for (int cc = c0 + lane; cc <= c1; cc += 32) state_merge(s, a.part[cc + b], c);
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        RowState o2 = state_shfl_xor(s, o);
        // keep the lower-lane state first so ties resolve to the lower index
        if (lane & o) { RowState t = o2; o2 = s; s = t; }
        state_merge(s, o2, c);
    }
    if (lane != 0) return;
    const RowState& t = s;
    const float* row = a.logits + (long long)b * a.ld;
    uint32_t err = bad_T ? ETI_ERRF_BAD_TEMP : 0u;
    if (!err) {
        if (t.m == -kInf) err = ETI_ERRF_ALL_NEG_INF;
        else if (t.m == kInf || isnan(t.S) || isnan(t.U)) err = ETI_ERRF_NONFINITE;
    }
    const float tau_in = a.tau[b];
    if (err) {
        a.tok[b] = -1;
        a.H[b] = __int_as_float(0x7fc00000);
        a.T_out[b] = Tt;
        if (a.dH) a.dH[b] = __int_as_float(0x7fc00000);
        if (a.theta_next) a.theta_next[b] = 0.f;
        if (a.surprisal) a.surprisal[b] = __int_as_float(0x7fc00000);
    } else {
        const float l2S = log2f(t.S);
        const float H = fmaxf(kLn2 * (l2S - t.U / t.S), 0.f);
        const float dH = a.H_prev[b] - H;
        a.tau[b] = tau_in + fmaxf(dH, 0.f);
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
        if (a.surprisal || a.surp_store) {
            const float tt = fmaf(row[t.bi], c, -t.mc);
            const float sp = kLn2 * (l2S - tt);
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
    a.share = (total + ncta - 1) / ncta;
    a.part = static_cast<RowState*>(part);
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
