// entropy_sample.cu -- half (a) of the entropic-time decode step:
// entropy H_t of softmax(z / T_t) (Section 2.1), entropy flow and entropic
// time (Section 2), the temperature law (Section 3.3), the next pruning
// threshold (Section 3.2 safety floor, Section 5 entropy floor) and a
// Gumbel-max draw from p_t, in ONE pass over the fp32 logits.
//
// Decomposition: a thread-block cluster of S CTAs per row; each CTA streams a
// contiguous chunk of the row with 128-bit loads and keeps, per thread, the
// online state
//     m  = running max of z          (raw logit units)
//     S  = sum 2^{t},  t = (z - m) * log2(e) / T
//     U  = sum 2^{t} * t
//     race best (w, E, index)  for the exponential race below.
// The CTA partials are merged through distributed shared memory by cluster
// rank 0, which writes the per-row outputs.  H = ln2 * (log2 S - U / S).
//
// Sampling.  argmax_x y_x - log(-log u_x) is argmax_x w_x / E_x with
// w_x = exp(y_x - m) and the exponential variate E_x = -log u_x, so the
// exp() already needed for S is reused and one log per token remains.
// Candidates are compared by cross-multiplication (w_a E_b > w_b E_a).
// E is computed in log2 units (the common factor cancels in the race):
//   u <= 15/16 : E2 = -lg2(u) with the MUFU approximation (|lg2 u| >= 0.093,
//                so its absolute error stays a small relative error);
//   u >  15/16 : v = 1 - u (exact), E2 = log2(e) * v * (1 + v/2 + ... + v^5/6),
//                the Taylor series of -log(1 - v), whose remainder is below
//                v^6/7 < 2^-24 / 7 relative.
// u = (2 (word >> 9) + 1) / 2^24 is formed exactly as (1.m - (1 - 2^-24)).
#include <cooperative_groups.h>

#include "common.cuh"

namespace cg = cooperative_groups;

namespace eti {

// Philox4x32-10 (Salmon et al., SC'11): ten rounds of two 32x32->64-bit
// multiplies; the key is bumped by the Weyl constants between rounds.
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        const unsigned long long p0 = (unsigned long long)0xD2511F53u * c.x;
        const unsigned long long p1 = (unsigned long long)0xCD9E8D57u * c.z;
        const uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
        const uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
        c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
        k0 += 0x9E3779B9u;
        k1 += 0xBB67AE85u;
    }
    return c;
}

// Exponential variate E / ln 2 from one 32-bit word (see the file comment).
__device__ __forceinline__ float exp_variate_log2(uint32_t word) {
    const float one_m = __uint_as_float((word >> 9) | 0x3F800000u);   // 1 + j 2^-23
    const float u = one_m - __uint_as_float(0x3F7FFFFFu);             // (2j + 1) 2^-24, exact
    const float v = 1.0f - u;                                         // exact for u > 1/2
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
    float S;    // sum 2^t
    float U;    // sum 2^t * t
    float bw;   // race best: w relative to m
    float bE;   // race best: E / ln 2
    int bi;     // race best: token index (INT_MAX = none)
};

__device__ __forceinline__ void state_init(RowState& s) {
    s.m = -kInf; s.S = 0.f; s.U = 0.f; s.bw = 0.f; s.bE = 1.f; s.bi = 0x7fffffff;
}

// Move the state to a new, larger reference max `nm`.
__device__ __forceinline__ void state_rebase(RowState& s, float nm, float c) {
    float a = 0.f, d = 0.f;
    if (s.m != -kInf) {
        d = (s.m - nm) * c;
        a = fast_ex2(d);
    }
    s.U = a * fmaf(d, s.S, s.U);
    s.S *= a;
    s.bw *= a;
    s.m = nm;
}

// Merge partial `o` into `s` (both may be empty).
__device__ __forceinline__ void state_merge(RowState& s, RowState o, float c) {
    const float nm = fmaxf(s.m, o.m);
    if (nm == -kInf) return;
    state_rebase(s, nm, c);
    state_rebase(o, nm, c);
    s.S += o.S;
    s.U += o.U;
    const float lhs = o.bw * s.bE, rhs = s.bw * o.bE;
    if (lhs > rhs || (lhs == rhs && o.bi < s.bi)) {
        s.bw = o.bw; s.bE = o.bE; s.bi = o.bi;
    }
}

__device__ __forceinline__ RowState state_shfl_xor(const RowState& s, int o) {
    RowState r;
    r.m = __shfl_xor_sync(0xffffffffu, s.m, o);
    r.S = __shfl_xor_sync(0xffffffffu, s.S, o);
    r.U = __shfl_xor_sync(0xffffffffu, s.U, o);
    r.bw = __shfl_xor_sync(0xffffffffu, s.bw, o);
    r.bE = __shfl_xor_sync(0xffffffffu, s.bE, o);
    r.bi = __shfl_xor_sync(0xffffffffu, s.bi, o);
    return r;
}

// One token: entropy sums and the race.
__device__ __forceinline__ void consume(RowState& s, float z, uint32_t word, int x, float c) {
    const float t = (z - s.m) * c;
    const float w = fast_ex2(t);
    s.S += w;
    s.U = fmaf(w, fmaxf(t, -250.f), s.U);   // -inf logits add 0 (w = 0); NaN still reaches S
    const float E = exp_variate_log2(word);
    if (w * s.bE > s.bw * E) { s.bw = w; s.bE = E; s.bi = x; }
}

constexpr int kEtsThreads = 256;
constexpr int kEtsBatch = 4;    // groups of 4 tokens loaded per thread per step

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
    int32_t* tok;
    float* H;
    float* T_out;
    float* dH;
    float* theta_next;
    float* surprisal;
    uint32_t* err;
    int groups_per_cta;   // groups of 4 tokens per cluster rank
};

template <bool kVec>
__global__ void __launch_bounds__(kEtsThreads)
entropy_temp_sample_kernel(const EtsArgs a) {
    cg::cluster_group cluster = cg::this_cluster();
    const int rank = (int)cluster.block_rank();
    const int nrank = (int)cluster.num_blocks();
    const int b = blockIdx.y;
    const int tid = threadIdx.x;
    __shared__ RowState warp_part[kEtsThreads / 32];
    __shared__ RowState cta_part;

    const float T = a.T_in[b];
    const bool bad_T = !(T > 0.f && T < kInf);
    const float c = bad_T ? 0.f : kLog2e / T;
    const float* row = a.logits + (long long)b * a.ld;
    const int ngroups = (a.V + 3) >> 2;
    const int g0 = min(rank * a.groups_per_cta, ngroups);
    const int g1 = min(g0 + a.groups_per_cta, ngroups);
    const int full_groups = a.V >> 2;   // groups with 4 in-range tokens

    RowState s;
    state_init(s);
    if (!bad_T) {
        for (int base = g0; base < g1; base += kEtsBatch * kEtsThreads) {
            float z[kEtsBatch][4];
#pragma unroll
            for (int k = 0; k < kEtsBatch; ++k) {
                const int g = base + k * kEtsThreads + tid;
                if (g < g1 && kVec && g < full_groups) {
                    const float4 v = ldg_stream_f4(row + 4 * (long long)g);
                    z[k][0] = v.x; z[k][1] = v.y; z[k][2] = v.z; z[k][3] = v.w;
                } else {
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int x = 4 * g + e;
                        z[k][e] = (g < g1 && x < a.V) ? __ldg(row + x) : -kInf;
                    }
                }
            }
            float bm = -kInf;
#pragma unroll
            for (int k = 0; k < kEtsBatch; ++k)
#pragma unroll
                for (int e = 0; e < 4; ++e) bm = fmaxf(bm, z[k][e]);
            if (bm == -kInf) {
                // every token of the batch is -inf (or NaN): nothing to add and
                // nothing to draw, but a NaN must still poison the row
                bool nan = false;
#pragma unroll
                for (int k = 0; k < kEtsBatch; ++k)
#pragma unroll
                    for (int e = 0; e < 4; ++e) nan |= (z[k][e] != z[k][e]);
                if (nan) s.S = __int_as_float(0x7fc00000);
                continue;
            }
            if (bm > s.m) state_rebase(s, bm, c);
#pragma unroll
            for (int k = 0; k < kEtsBatch; ++k) {
                const int g = base + k * kEtsThreads + tid;
                if (g < g1) {
                    const uint4 r = philox4x32_10(make_uint4((uint32_t)g, (uint32_t)b, a.off_lo, a.off_hi),
                                                  a.seed_lo, a.seed_hi);
                    consume(s, z[k][0], r.x, 4 * g + 0, c);
                    consume(s, z[k][1], r.y, 4 * g + 1, c);
                    consume(s, z[k][2], r.z, 4 * g + 2, c);
                    consume(s, z[k][3], r.w, 4 * g + 3, c);
                }
            }
        }
    }
    // CTA reduction: warp shuffles, then one warp over the warp partials.
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) state_merge(s, state_shfl_xor(s, o), c);
    if ((tid & 31) == 0) warp_part[tid >> 5] = s;
    __syncthreads();
    if (tid == 0) {
        RowState t = warp_part[0];
        for (int w = 1; w < kEtsThreads / 32; ++w) state_merge(t, warp_part[w], c);
        cta_part = t;
    }
    cluster.sync();
    if (rank == 0 && tid == 0) {
        RowState t = cta_part;
        for (int r = 1; r < nrank; ++r) state_merge(t, *cluster.map_shared_rank(&cta_part, r), c);
        uint32_t err = bad_T ? ETI_ERRF_BAD_TEMP : 0u;
        if (!err) {
            if (t.m == -kInf) err = ETI_ERRF_ALL_NEG_INF;
            else if (t.m == kInf || isnan(t.S) || isnan(t.U)) err = ETI_ERRF_NONFINITE;
        }
        const float tau_in = a.tau[b];
        if (err) {
            a.tok[b] = -1;
            a.H[b] = __int_as_float(0x7fc00000);
            a.T_out[b] = T;
            if (a.dH) a.dH[b] = __int_as_float(0x7fc00000);
            if (a.theta_next) a.theta_next[b] = 0.f;
            if (a.surprisal) a.surprisal[b] = __int_as_float(0x7fc00000);
        } else {
            const float l2S = log2f(t.S);
            const float H = fmaxf(kLn2 * (l2S - t.U / t.S), 0.f);
            const float dH = a.H_prev[b] - H;
            a.tau[b] = tau_in + fmaxf(dH, 0.f);
            float Tn = T * expf(a.p.sign * a.p.eta * (H - a.H_target[b]));
            Tn = fminf(a.p.T_max, fmaxf(a.p.T_min, Tn));
            a.tok[b] = t.bi;
            a.H[b] = H;
            a.T_out[b] = Tn;
            if (a.dH) a.dH[b] = dH;
            if (a.theta_next) {
                const float Heff = fmaxf(H - a.p.eps_H, a.p.H_min);
                const float tmax = a.V > 1 ? a.p.theta_hi * fmaxf(0.f, 1.f - Heff / logf((float)a.V))
                                           : a.p.theta_hi;
                a.theta_next[b] = fminf(a.p.theta_user, tmax);
            }
            if (a.surprisal) {
                const float tt = (row[t.bi] - t.m) * c;
                a.surprisal[b] = kLn2 * (l2S - tt);
            }
        }
        a.err[b] = err;
    }
    // keep every CTA's shared memory alive until rank 0 has read it
    cluster.sync();
}

}  // namespace eti

// Host launcher (called from the C ABI after argument validation).
int eti_launch_entropy_temp_sample(const float* logits, int B, int V, long long ld,
                                   const float* T_in, const float* H_prev, float* tau,
                                   const float* H_target, const eti_ctrl_params* p,
                                   uint64_t seed, uint64_t offset, int32_t* tok, float* H,
                                   float* T_out, float* dH, float* theta_next, float* surprisal,
                                   uint32_t* err, cudaStream_t stream, int cluster_override) {
    using namespace eti;
    if (B == 0) return ETI_OK;
    const int ngroups = (V + 3) / 4;
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    // aim for ~4 CTAs per SM in one wave, at least one group per thread
    int S = cluster_override > 0 ? cluster_override : 1;
    if (cluster_override <= 0) {
        const int want = ceil_div(4 * sms, B);
        const int cap = max(1, ceil_div(ngroups, kEtsThreads));
        while (S < 8 && S < want && S < cap) S <<= 1;
    }
    EtsArgs a;
    a.logits = logits; a.B = B; a.V = V; a.ld = ld; a.T_in = T_in; a.H_prev = H_prev;
    a.tau = tau; a.H_target = H_target; a.p = *p;
    a.seed_lo = (uint32_t)seed; a.seed_hi = (uint32_t)(seed >> 32);
    a.off_lo = (uint32_t)offset; a.off_hi = (uint32_t)(offset >> 32);
    a.tok = tok; a.H = H; a.T_out = T_out; a.dH = dH; a.theta_next = theta_next;
    a.surprisal = surprisal; a.err = err;
    a.groups_per_cta = ceil_div(ngroups, S);
    const bool vec = (ld % 4 == 0) && ((reinterpret_cast<uintptr_t>(logits) & 15) == 0);

    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(S, B, 1);
    cfg.blockDim = dim3(kEtsThreads, 1, 1);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = S;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t e = vec ? cudaLaunchKernelEx(&cfg, entropy_temp_sample_kernel<true>, a)
                        : cudaLaunchKernelEx(&cfg, entropy_temp_sample_kernel<false>, a);
    return e == cudaSuccess ? ETI_OK : ETI_ERR_CUDA;
}
