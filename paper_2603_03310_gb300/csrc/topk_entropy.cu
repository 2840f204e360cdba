// topk_entropy.cu -- the top-k entropy estimators of Section 2.1.
//
// With y = z / T_t, p = softmax(y) and K the first k tokens ordered by
// (y descending, token id ascending):
//   H~ = -sum_{x in K} p~(x) log p~(x),  p~ = p / sum_K p      (truncated)
//   m_bar = sum_{x not in K} p(x)                              (tail mass)
//   H^ = H~ + h(m_bar) + m_bar log(V - k)                      (tail-corrected)
//
// Only the VALUES of K matter: tokens tied at the k-th key contribute the same
// amount whichever of them the (token id) rule picks, so the kernel needs the
// k-th largest logit and how many of its ties belong to K, not the set.  One
// CTA per row finds them.  The first pass takes the row max, checks for NaN /
// +inf and keeps each thread's own max; when k <= threads, the k-th largest of
// those maxima is a lower bound tau of the k-th largest logit (at least k
// tokens reach it), so only the tokens >= tau are candidates: they are
// gathered in shared memory by a second pass and sorted (bitonic).  When k is
// larger or the candidates overflow, a radix select on the order-preserving
// 32-bit key of the logit (11 + 11 + 10 bits) finds the k-th key instead.
// A last pass forms, in base 2 against the max,
//   Z_K = sum_{K} 2^t,  U_K = sum_{K} 2^t t,  Z_tail = sum_{not K} 2^t,
// with the tokens at the max counted (each adds exactly 1) so that a
// near-deterministic K keeps its precision.  The first pass reads the row
// from HBM, the others from L2.  Histogram updates are warp-aggregated
// (one shared-memory atomic per distinct bin per warp).
#include "common.cuh"

namespace eti {

constexpr int kTkThreads = 512;
constexpr int kTkWarps = kTkThreads / 32;
constexpr int kTkCand = 4096;       // candidate keys of the fast path

struct TkArgs {
    const float* logits;
    int B, V;
    long long ld;
    const float* T_in;
    int k;
    float* H_tilde;
    float* H_hat;
    float* tail_mass;     // nullable
    uint32_t* err;
};

// order-preserving key of an fp32 value (NaN never reaches the ordering)
__device__ __forceinline__ uint32_t tk_key(float f) {
    const uint32_t b = __float_as_uint(f);
    return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float tk_value(uint32_t key) {
    return __uint_as_float((key & 0x80000000u) ? (key & 0x7FFFFFFFu) : ~key);
}

// hist[bin] += 1 for the lanes with `on`, one atomic per distinct bin
__device__ __forceinline__ void tk_hist_add(uint32_t* hist, uint32_t bin, bool on) {
    const uint32_t act = __ballot_sync(0xffffffffu, on);
    if (on) {
        const uint32_t peers = __match_any_sync(act, bin);
        if ((threadIdx.x & 31) == __ffs(peers) - 1) atomicAdd(hist + bin, (uint32_t)__popc(peers));
    }
}

// The bin (counted from the top) where the running count reaches `need`, and
// the count still needed inside it; one warp scans, the CTA reads the result.
__device__ __forceinline__ void tk_find(const uint32_t* hist, int nbins, int need, int* sel) {
    __syncthreads();
    if (threadIdx.x < 32) {
        const int lane = threadIdx.x, per = nbins / 32;
        const int top = nbins - 1 - lane * per;           // this lane: bins top, top-1, ..., top-per+1
        uint32_t s = 0;
        for (int i = 0; i < per; ++i) s += hist[top - i];
        uint32_t incl = s;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += y;
        }
        const uint32_t above = incl - s;
        if ((int)above < need && need <= (int)incl) {
            int acc = (int)above;
            for (int i = 0; i < per; ++i) {
                const int c = (int)hist[top - i];
                if (need <= acc + c) { sel[0] = top - i; sel[1] = need - acc; break; }
                acc += c;
            }
        }
    }
    __syncthreads();
}

// Sort s[0..n) descending in shared memory (bitonic network, n a power of 2).
__device__ __forceinline__ void tk_sort_desc(uint32_t* s, int n) {
    for (int size = 2; size <= n; size <<= 1)
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            for (int p = threadIdx.x; p < (n >> 1); p += kTkThreads) {
                const int i = (p / stride) * 2 * stride + (p % stride), l = i + stride;
                const uint32_t x = s[i], y = s[l];
                if (((i & size) == 0) == (x < y)) { s[i] = y; s[l] = x; }
            }
            __syncthreads();
        }
}

template <int N>
__device__ __forceinline__ void tk_block_sum(float (&v)[N], float* red) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
#pragma unroll
    for (int i = 0; i < N; ++i) v[i] = warp_sum(v[i]);
    __syncthreads();
    if (lane == 0)
#pragma unroll
        for (int i = 0; i < N; ++i) red[i * kTkWarps + w] = v[i];
    __syncthreads();
#pragma unroll
    for (int i = 0; i < N; ++i) {
        float r = 0.f;
        for (int u = 0; u < kTkWarps; ++u) r += red[i * kTkWarps + u];   // fixed order
        v[i] = r;
    }
}

// Visit every element of the row (all threads run the same number of steps,
// so the warp collectives inside `f` see full warps); f(z, valid).  Each
// step issues eight independent 16-byte loads per thread before using them.
template <bool kVec, typename F>
__device__ __forceinline__ void tk_row(const float* row, int V, F&& f) {
    constexpr int U = 8;
    const int tid = threadIdx.x;
    for (int base = 0; base < V; base += 4 * kTkThreads * U) {
        float z[U][4];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int x = base + 4 * (u * kTkThreads + tid);
            if (kVec && x + 3 < V) {
                const float4 v = __ldg(reinterpret_cast<const float4*>(row + x));
                z[u][0] = v.x; z[u][1] = v.y; z[u][2] = v.z; z[u][3] = v.w;
            } else {
#pragma unroll
                for (int e = 0; e < 4; ++e) z[u][e] = x + e < V ? __ldg(row + x + e) : 0.f;
            }
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int x = base + 4 * (u * kTkThreads + tid);
#pragma unroll
            for (int e = 0; e < 4; ++e) f(z[u][e], x + e < V);
        }
    }
}

template <bool kVec>
__global__ void __launch_bounds__(kTkThreads) topk_entropy_kernel(const TkArgs a) {
    pdl_trigger();
    pdl_wait();
    __shared__ uint32_t hist[2048];
    __shared__ uint32_t cand[kTkCand];
    __shared__ float red[4 * kTkWarps];
    __shared__ int sel[2];
    __shared__ int ncand;
    const int b = blockIdx.x, tid = threadIdx.x;
    const float T = a.T_in[b];
    const bool bad_T = !(T > 0.f && T < kInf);
    const float c = bad_T ? 0.f : kLog2e / T;
    const float* row = a.logits + (long long)b * a.ld;
    const int V = a.V, ke = min(a.k, V);

    // pass 1: row max, NaN / +inf, each thread's own max
    float zmax = -kInf;
    int nonfin = 0;
    tk_row<kVec>(row, V, [&](float z, bool on) {
        if (on) {
            nonfin |= (z != z) || (z == kInf);
            zmax = fmaxf(zmax, z);
        }
    });
    const float lmax = zmax;
    zmax = warp_max(zmax);
    if ((tid & 31) == 0) red[tid >> 5] = zmax;
    const int any_nonfin = __syncthreads_or(nonfin);
    float m = -kInf;
    for (int u = 0; u < kTkWarps; ++u) m = fmaxf(m, red[u]);
    uint32_t err = bad_T ? ETI_ERRF_BAD_TEMP : 0u;
    if (!err && any_nonfin) err = ETI_ERRF_NONFINITE;
    if (!err && m == -kInf) err = ETI_ERRF_ALL_NEG_INF;
    if (err) {
        if (tid == 0) {
            const float nan = __int_as_float(0x7fc00000);
            a.H_tilde[b] = nan;
            a.H_hat[b] = nan;
            if (a.tail_mass) a.tail_mass[b] = nan;
            a.err[b] = err;
        }
        return;
    }

    const uint32_t kmax = tk_key(m);
    const float mc = m * c;
    // per thread: Z_K below the max, U_K, Z_tail, tokens at the max inside K
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    bool fast = ke <= kTkThreads;
    if (fast) {
        // tau: the ke-th largest thread maximum; at least ke tokens are >= tau
        cand[tid] = tk_key(lmax);                  // -inf for a thread with no token
        __syncthreads();
        tk_sort_desc(cand, kTkThreads);
        const uint32_t tau = cand[ke - 1];
        if (tid == 0) ncand = 0;
        __syncthreads();
        // tokens below tau are in the tail whatever K is: sum them here
        float zt = 0.f;
        tk_row<kVec>(row, V, [&](float z, bool on) {
            if (!on) return;
            const uint32_t key = tk_key(z);
            if (key >= tau) {
                const int i = atomicAdd(&ncand, 1);
                if (i < kTkCand) cand[i] = key;
            } else {
                zt += fast_ex2(fmaf(z, c, -mc));
            }
        });
        __syncthreads();
        const int n = ncand;
        fast = n <= kTkCand;                       // uniform
        if (fast) {
            int np2 = 1;
            while (np2 < n) np2 <<= 1;
            for (int i = n + tid; i < np2; i += kTkThreads) cand[i] = 0u;   // below every key
            __syncthreads();
            tk_sort_desc(cand, np2);
            // K = the first ke candidates (tied values contribute alike whichever
            // of them the token-id rule picks); the others join the tail
            for (int i = tid; i < n; i += kTkThreads) {
                const uint32_t key = cand[i];
                if (key == kmax) {
                    if (i < ke) acc[3] += 1.f; else zt += 1.f;
                } else {
                    const float t = fmaf(tk_value(key), c, -mc);
                    const float w = fast_ex2(t);
                    if (i < ke) {
                        acc[0] += w;
                        acc[1] = fmaf(w, fmaxf(t, -250.f), acc[1]);   // -inf logits add 0
                    } else {
                        zt += w;
                    }
                }
            }
            acc[2] = zt;
        }
    }
    if (!fast) {
        // radix select of the k-th largest key: 11 + 11 + 10 bits
        for (int i = tid; i < 2048; i += kTkThreads) hist[i] = 0;
        __syncthreads();
        tk_row<kVec>(row, V, [&](float z, bool on) { tk_hist_add(hist, tk_key(z) >> 21, on); });
        tk_find(hist, 2048, ke, sel);
        const uint32_t b0 = (uint32_t)sel[0];
        int need = sel[1];
        for (int i = tid; i < 2048; i += kTkThreads) hist[i] = 0;
        __syncthreads();
        tk_row<kVec>(row, V, [&](float z, bool on) {
            const uint32_t key = tk_key(z);
            tk_hist_add(hist, (key >> 10) & 2047u, on && (key >> 21) == b0);
        });
        tk_find(hist, 2048, need, sel);
        const uint32_t b1 = (uint32_t)sel[0];
        need = sel[1];
        for (int i = tid; i < 2048; i += kTkThreads) hist[i] = 0;
        __syncthreads();
        const uint32_t pre = (b0 << 11) | b1;
        tk_row<kVec>(row, V, [&](float z, bool on) {
            const uint32_t key = tk_key(z);
            tk_hist_add(hist, key & 1023u, on && (key >> 10) == pre);
        });
        tk_find(hist, 1024, need, sel);
        const uint32_t kth = (pre << 10) | (uint32_t)sel[0];
        const int rem = sel[1];                    // ties at the k-th key that belong to K
        // sums against the max (base 2): tokens at the max are counted, not summed
        float v[4] = {0.f, 0.f, 0.f, 0.f};        // Z_K (below the max), U_K, Z_tail, #at the k-th key
        int ntop = 0;
        tk_row<kVec>(row, V, [&](float z, bool on) {
            if (!on) return;
            const uint32_t key = tk_key(z);
            if (key == kmax) { ++ntop; return; }
            const float t = fmaf(z, c, -mc);
            const float w = fast_ex2(t);
            if (key > kth) {
                v[0] += w;
                v[1] = fmaf(w, fmaxf(t, -250.f), v[1]);   // -inf logits add 0
            } else if (key < kth) {
                v[2] += w;
            } else {
                v[3] += 1.f;
            }
        });
        tk_block_sum<4>(v, red);
        float nt[1] = {(float)ntop};
        __syncthreads();
        tk_block_sum<1>(nt, red);
        // the rem tokens at the k-th key join K, the others the tail
        if (kth == kmax) {
            acc[3] = (float)rem;                   // K = rem of the tokens at the max
            acc[2] = v[2] + nt[0] - (float)rem;
            acc[0] = v[0];
            acc[1] = v[1];
        } else {
            const float tk = fmaf(tk_value(kth), c, -mc);
            const float wk = fast_ex2(tk);
            acc[3] = nt[0];
            acc[0] = fmaf((float)rem, wk, v[0]);
            acc[1] = fmaf((float)rem * wk, fmaxf(tk, -250.f), v[1]);
            acc[2] = fmaf(v[3] - (float)rem, wk, v[2]);
        }
    } else {
        tk_block_sum<4>(acc, red);
    }

    if (tid != 0) return;
    const float ZKr = acc[0], UK = acc[1], Zt = acc[2], nK = acc[3];   // nK >= 1: the max is in K
    const float ZK = nK + ZKr;
    const float lnZK = logf(nK) + log1pf(ZKr / nK);
    const float Ht = fmaxf(lnZK - kLn2 * UK / ZK, 0.f);
    const float mb = Zt / (ZK + Zt);
    float hb = 0.f;
    if (mb > 0.f && mb < 1.f) hb = -mb * logf(mb) - (1.f - mb) * log1pf(-mb);
    a.H_tilde[b] = Ht;
    a.H_hat[b] = Ht + hb + (ke < V ? mb * logf((float)(V - ke)) : 0.f);
    if (a.tail_mass) a.tail_mass[b] = mb;
    a.err[b] = 0u;
}

}  // namespace eti

using namespace eti;

int eti_launch_topk_entropy(const float* logits, int B, int V, long long ld, const float* T_in,
                            int k, float* H_tilde, float* H_hat, float* tail_mass, uint32_t* err,
                            cudaStream_t stream) {
    if (B == 0) return ETI_OK;
    TkArgs a;
    a.logits = logits; a.B = B; a.V = V; a.ld = ld; a.T_in = T_in; a.k = k;
    a.H_tilde = H_tilde; a.H_hat = H_hat; a.tail_mass = tail_mass; a.err = err;
    const bool vec = (ld % 4 == 0) && ((reinterpret_cast<uintptr_t>(logits) & 15) == 0);
    const cudaError_t e = vec ? eti_launch_pdl(topk_entropy_kernel<true>, dim3(B), dim3(kTkThreads), 0, stream, a)
                              : eti_launch_pdl(topk_entropy_kernel<false>, dim3(B), dim3(kTkThreads), 0, stream, a);
    return e == cudaSuccess ? ETI_OK : ETI_ERR_CUDA;
}
