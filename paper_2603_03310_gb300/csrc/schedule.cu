// schedule.cu -- entropy-aware scheduling priority and admission (Section 3.1).
//
//   E[dH_s] <- lambda E[dH_s] + (1 - lambda) max(0, dH_s)   (a NaN dH leaves it)
//   pi(s)    = E[dH_s] / max(alpha C_s + beta M_s + gamma L_s, den_min)
// with C_s the kept tokens per kv head, M_s the context length and L_s the
// caller's urgency; the `budget` sequences of highest pi are admitted (ties to
// the lower index, NaN below every number).  One CTA: each thread owns a
// contiguous range of sequences; the admitted set is a radix select on the
// order-preserving key of pi (4 x 8 bits) plus an index-ordered rank of the
// ties at the cut.
#include "common.cuh"

namespace eti {

constexpr int kSchThreads = 1024;
constexpr int kSchWarps = kSchThreads / 32;

struct SchArgs {
    const float* dH;
    float* ema;
    const int32_t* kept_cnt;   // [B][Hkv] or null
    int Hkv, P;
    const int32_t* ctx_lens;   // or null
    const float* urgency;      // or null
    eti_sched_params p;
    int B, budget;
    float* priority;
    uint8_t* admit;
};

__device__ __forceinline__ uint32_t sch_key(float f) {
    if (f != f) return 0u;                        // NaN below every number
    const uint32_t b = __float_as_uint(f);
    return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

__global__ void __launch_bounds__(kSchThreads) schedule_kernel(const SchArgs a) {
    pdl_trigger();
    pdl_wait();
    __shared__ int hist[256];
    __shared__ int wsum[kSchWarps];
    __shared__ int sel_digit, sel_rem;
    const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
    const int per = (a.B + kSchThreads - 1) / kSchThreads;
    const int s0 = min(tid * per, a.B), s1 = min(s0 + per, a.B);

    // priorities
    for (int s = s0; s < s1; ++s) {
        const float d = a.dH[s];
        float e = a.ema[s];
        if (d == d) e = fmaf(a.p.lambda, e, (1.f - a.p.lambda) * fmaxf(0.f, d));
        float C = 0.f;
        if (a.kept_cnt) {
            int kc = 0;
            for (int h = 0; h < a.Hkv; ++h) kc += a.kept_cnt[(long long)s * a.Hkv + h];
            C = (float)kc * (float)a.P / (float)a.Hkv;
        }
        const float M = a.ctx_lens ? (float)a.ctx_lens[s] : 0.f;
        const float L = a.urgency ? a.urgency[s] : 0.f;
        const float den = fmaxf(fmaf(a.p.alpha, C, fmaf(a.p.beta, M, a.p.gamma * L)), a.p.den_min);
        a.ema[s] = e;
        a.priority[s] = e / den;
    }
    __syncthreads();   // this thread's priorities are re-read below (same thread; order only)

    const int n = min(max(a.budget, 0), a.B);
    uint32_t kth = 0u;
    int rem = 0;
    if (n > 0 && n < a.B) {
        // radix select of the n-th largest key, 8 bits at a time
        uint32_t prefix = 0, mask = 0;
        int need = n;
        for (int digit = 3; digit >= 0; --digit) {
            const int sh = digit * 8;
            for (int i = tid; i < 256; i += kSchThreads) hist[i] = 0;
            __syncthreads();
            for (int s = s0; s < s1; ++s) {
                const uint32_t key = sch_key(a.priority[s]);
                if ((key & mask) == prefix) atomicAdd(&hist[(key >> sh) & 255], 1);
            }
            __syncthreads();
            if (tid < 32) {
                int cnt8[8], s8 = 0;
#pragma unroll
                for (int e = 0; e < 8; ++e) { cnt8[e] = hist[255 - (tid * 8 + e)]; s8 += cnt8[e]; }
                int incl = s8;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const int y = __shfl_up_sync(0xffffffffu, incl, o);
                    if (tid >= o) incl += y;
                }
                int above = incl - s8;
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    if (above < need && need <= above + cnt8[e]) {
                        sel_digit = 255 - (tid * 8 + e);
                        sel_rem = need - above;
                    }
                    above += cnt8[e];
                }
            }
            __syncthreads();
            prefix |= (uint32_t)sel_digit << sh;
            mask |= 255u << sh;
            need = sel_rem;
            __syncthreads();
        }
        kth = prefix;
        rem = need;
    }
    // ties at the cut in index order: exclusive scan of each thread's tie count
    int eq = 0;
    if (n > 0 && n < a.B)
        for (int s = s0; s < s1; ++s) eq += sch_key(a.priority[s]) == kth;
    int x = eq;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) wsum[w] = x;
    __syncthreads();
    int rank = x - eq;
    for (int i = 0; i < w; ++i) rank += wsum[i];
    for (int s = s0; s < s1; ++s) {
        bool in;
        if (n <= 0) in = false;
        else if (n >= a.B) in = true;
        else {
            const uint32_t key = sch_key(a.priority[s]);
            in = key > kth;
            if (key == kth) in = rank++ < rem;
        }
        a.admit[s] = in ? 1 : 0;
    }
}

}  // namespace eti

using namespace eti;

int eti_launch_schedule(const float* dH, float* ema, const int32_t* kept_cnt, int Hkv, int P,
                        const int32_t* ctx_lens, const float* urgency, const eti_sched_params* p,
                        int B, int budget, float* priority, uint8_t* admit, cudaStream_t stream) {
    if (B == 0) return ETI_OK;
    SchArgs a;
    a.dH = dH; a.ema = ema; a.kept_cnt = kept_cnt; a.Hkv = Hkv; a.P = P; a.ctx_lens = ctx_lens;
    a.urgency = urgency; a.p = *p; a.B = B; a.budget = budget; a.priority = priority; a.admit = admit;
    return eti_launch_pdl(schedule_kernel, dim3(1), dim3(kSchThreads), 0, stream, a) == cudaSuccess
               ? ETI_OK : ETI_ERR_CUDA;
}
