// keep_set.cuh -- shared pieces of the keep-set kernels (Section 3.2: block
// scores, the threshold / budget rule, compaction, the kept-token softmax
// normaliser): the argument block, the order-preserving key, and the
// per-head reductions and ranks of the flat layout (thread t owns query head
// t % GP of its blocks).
#pragma once

#include "common.cuh"

namespace eti {

struct FinArgs {
    const float4* stats;
    const int32_t* ctx_lens;
    const int32_t* block_table;
    long long num_pages;
    int B, Hq, Hkv, g, P, max_blocks;
    // rule mode (given == 0)
    const float* theta;
    int B_min;
    int score_mode;         // 0 A: I_i = -log a_i; 1 E: stored surprisal; 2 M: 1
    // given mode: keep set from a list or a mask (or every block)
    int given;
    const uint8_t* given_mask;
    const int32_t* given_idx;
    const int32_t* given_cnt;
    // outputs
    uint8_t* keep_mask;     // nullable
    int32_t* kept_idx;
    int32_t* kept_cnt;
    float* block_score;     // nullable
    float* kept_norm;       // nullable: [B][Hq][2]
    uint32_t* err;          // nullable
    int share_cache;        // wide kernel with the term cache: also cache each
                            // block-head's share (1 + l1) e^{m - M} of Z
};

// e^d for d <= 0 (a block's weight against the head's max) with the MUFU
// exp2: relative error about 2^-22 plus |d| 2^-24 from the scaling, far below
// the 1e-5 keep-decision ties; weights below 2^-126 flush to zero.
__device__ __forceinline__ float exp_le0(float d) { return fast_ex2(d * kLog2e); }

__device__ __forceinline__ uint32_t order_key(float f) {
    if (f != f) return 0u;
    const uint32_t b = __float_as_uint(f);
    return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

constexpr int kFlatPer = 16;
constexpr int kWideThreads = 1024;
constexpr size_t kWideSmemMax = 200 * 1024;   // dynamic shared memory of the cached-term variant

template <int G>
struct FlatGP { static constexpr int v = G <= 1 ? 1 : G <= 2 ? 2 : G <= 4 ? 4 : 8; };

// per-head reduction of N values over the lanes (and warps) of equal h;
// red holds N * 32 * GP floats and must not be reused before the next barrier
template <int GP, int N, bool kMax>
__device__ __forceinline__ void head_reduce(float (&v)[N], float* red) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
#pragma unroll
    for (int o = 16; o >= GP; o >>= 1)
#pragma unroll
        for (int i = 0; i < N; ++i) {
            const float y = __shfl_xor_sync(0xffffffffu, v[i], o);
            v[i] = kMax ? fmaxf(v[i], y) : v[i] + y;
        }
    if (lane < GP)
#pragma unroll
        for (int i = 0; i < N; ++i) red[(i * 32 + w) * GP + lane] = v[i];
    __syncthreads();
    const int h = lane & (GP - 1);
#pragma unroll
    for (int i = 0; i < N; ++i) {
        float r = kMax ? -kInf : 0.f;
        for (int u = 0; u < nw; ++u) {
            const float y = red[(i * 32 + u) * GP + h];
            r = kMax ? fmaxf(r, y) : r + y;
        }
        v[i] = r;
    }
}

// The same reduction in two stages, for CTAs of many warps: after the warps'
// partials are in `red`, warp u < GP reduces head u's partials over the warps
// (one load per lane, a shuffle butterfly) and publishes it in `fin`
// (N * GP floats), so that each thread reads one value per reduction instead of
// one per warp.  Two barriers.
template <int GP, int N, bool kMax>
__device__ __forceinline__ void head_reduce2(float (&v)[N], float* red, float* fin) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
#pragma unroll
    for (int o = 16; o >= GP; o >>= 1)
#pragma unroll
        for (int i = 0; i < N; ++i) {
            const float y = __shfl_xor_sync(0xffffffffu, v[i], o);
            v[i] = kMax ? fmaxf(v[i], y) : v[i] + y;
        }
    if (lane < GP)
#pragma unroll
        for (int i = 0; i < N; ++i) red[(i * 32 + w) * GP + lane] = v[i];
    __syncthreads();
    if (w < GP) {
#pragma unroll
        for (int i = 0; i < N; ++i) {
            float r = lane < nw ? red[(i * 32 + lane) * GP + w] : (kMax ? -kInf : 0.f);
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                const float y = __shfl_xor_sync(0xffffffffu, r, o);
                r = kMax ? fmaxf(r, y) : r + y;
            }
            if (lane == 0) fin[i * GP + w] = r;
        }
    }
    __syncthreads();
    const int h = lane & (GP - 1);
#pragma unroll
    for (int i = 0; i < N; ++i) v[i] = fin[i * GP + h];
}

// Exclusive ranks in ascending block order of the flagged blocks (flags
// agree across the GP lanes of a block); returns the number flagged.
// scan holds KP * 32 + 1 ints.
template <int GP, int KP = kFlatPer>
__device__ __forceinline__ int flat_ranks(const bool (&f)[KP], int (&pos)[KP], int* scan) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
    const bool lead = (lane & (GP - 1)) == 0;
    const uint32_t below = (1u << (lane & ~(GP - 1))) - 1u;   // lanes of earlier blocks
    uint32_t bal[KP];
#pragma unroll
    for (int k = 0; k < KP; ++k) {
        bal[k] = __ballot_sync(0xffffffffu, f[k] && lead);
        if (lane == 0) scan[k * nw + w] = __popc(bal[k]);
    }
    __syncthreads();
    if (w == 0) {
        // exclusive scan of the (chunk, warp) counts, chunk-major
        const int E = KP * nw, per = (E + 31) >> 5;
        const int e0 = min(lane * per, E), e1 = min(e0 + per, E);
        int s = 0;
        for (int e = e0; e < e1; ++e) s += scan[e];
        int x = s;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x += y;
        }
        int run = x - s;
        for (int e = e0; e < e1; ++e) { const int c = scan[e]; scan[e] = run; run += c; }
        if (lane == 31) scan[E] = x;
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < KP; ++k) pos[k] = scan[k * nw + w] + __popc(bal[k] & below);
    return scan[KP * nw];
}

}  // namespace eti
