// score_prune.cu -- entropic block scores and the keep set (Section 3.2).
//
// score_blocks (the HBM-bound pass): every key page chunk (page, kv head) is
// read exactly once.  Warps walk a flattened list of (sequence, kv head,
// block) units, each warp taking an equal contiguous share (no idle tail);
// a unit is P/16 tiles of 16 tokens x D.  Each warp streams its tiles through
// a private ring of shared-memory stages filled by the Tensor Memory
// Accelerator (one lane issues 2-D tiled copies of 64-element boxes with the
// 128-byte swizzle, completing on the stage's mbarrier; every wait is
// bounded and a stage that never arrives is reported as a timeout).  q.k^T
// runs on bf16 m16n8k16 tensor-core tiles (tokens = M, query heads of the
// GQA group = N, head_dim = K) read conflict-free from the swizzled stage.
// Per block and query head it emits the stats (m_b, l_b - 1, u_b, e_b) =
// (max x, sum e^{x-m_b} - 1 kept exact, sum e^{x-m_b}(x-m_b), and for score
// mode E sum e^{x-m_b} s_i) and, optionally, the scaled scores x_i
// themselves so the decode pass never reads a key page again.
//
// prune_finalize (one CTA per (sequence, kv head)): with M = max_b m_b and
// Z = sum_b l_b e^{m_b - M}, the block term of the attention entropy is
//   I_b = e^{m_b - M} [ l_b (log Z + M - m_b) - u_b ] / Z,
// which is sum_{i in b} a_i (-log a_i) with a_i = e^{x_i - M} / Z written
// over the block stats (both bracket terms are >= 0, so no cancellation).
// Then the normalised group score, the threshold, the B_min budget (radix
// select, ties to the lower block index), compaction, and the kept-token
// softmax normaliser (max, sum) that the decode pass uses.  This file holds
// the scorer and the keep-set entry; the keep-set kernels are in
// keep_tile.cu (segments of up to 8192 block-heads, rule mode) and
// prune_wide.cu (longer segments, and the given keep sets of a standalone
// decode).
#include "common.cuh"
#include "keep_set.cuh"

namespace eti {

constexpr int kScoreThreads = 256;
constexpr int kScoreWarps = kScoreThreads / 32;

struct ScoreArgs {
    const uint16_t* q;
    const uint16_t* k_cache;
    const int32_t* block_table;
    const int32_t* ctx_lens;
    int B, Hq, Hkv, g, max_blocks;
    long long num_pages;
    float scale;
    float* token_scores;   // [B][Hkv][max_blocks][P][g] or null
    float4* stats;         // [B][Hkv][max_blocks][g]: (m, l - 1, u, e) with
                           // e = sum e^{x-m} s_i when tok_surp is given, else 0
    const float* tok_surp; // [num_pages][P] stored token surprisal s_i, or null
    int wait_iters;        // polls before a tile wait gives up (eti_set_wait_limit)
};

// Exclusive prefix over sequences of (blocks * Hkv) into shared memory;
// returns the total.  cum has B + 1 entries.
__device__ int units_prefix(const int32_t* ctx_lens, int B, int P, int max_blocks, int Hkv,
                            int* cum, int* warp_tot) {
    const int tid = threadIdx.x, nt = blockDim.x;
    int carry = 0;
    for (int base = 0; base < B; base += nt) {
        const int b = base + tid;
        const int v = b < B ? seq_blocks(ctx_lens[b], P, max_blocks) * Hkv : 0;
        // block-wide inclusive scan
        int x = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, x, o);
            if ((tid & 31) >= o) x += y;
        }
        if ((tid & 31) == 31) warp_tot[tid >> 5] = x;
        __syncthreads();
        int wofs = 0, tot = 0;
        for (int w = 0; w < (nt >> 5); ++w) {
            if (w < (tid >> 5)) wofs += warp_tot[w];
            tot += warp_tot[w];
        }
        if (b < B) cum[b] = carry + wofs + x - v;
        carry += tot;
        __syncthreads();
    }
    if (tid == 0) cum[B] = carry;
    __syncthreads();
    return carry;
}

// Per-warp ring of TMA tiles (16 tokens x D bf16, 128-byte swizzle).
template <int D>
struct ScoreRing {
    static constexpr int kTile = 16 * D * 2;             // bytes of one 16-token tile
    static constexpr int kStages = D == 128 ? 3 : 5;     // tiles in flight per warp
};

template <int D, int P>
__host__ __device__ constexpr size_t score_smem_bytes(int B) {
    return 1024                                                                 // alignment slack
           + (size_t)kScoreWarps * ScoreRing<D>::kStages * ScoreRing<D>::kTile   // tiles
           + (size_t)kScoreWarps * ScoreRing<D>::kStages * 8                    // barriers
           + (size_t)kScoreWarps * 64 * 16                                      // unit tables
           + (((size_t)(B + 1) * 4 + 15) & ~size_t(15));                        // prefix
}

template <int D, int P>
__global__ void __launch_bounds__(kScoreThreads, 2)
score_blocks_kernel(const __grid_constant__ CUtensorMap kmap, const ScoreArgs a) {
    constexpr int kTiles = P / 16;
    constexpr int S = ScoreRing<D>::kStages;
    constexpr int TB = ScoreRing<D>::kTile;
    constexpr int H = D / 64;                    // 64-element boxes per tile row
    pdl_trigger();
    pdl_wait();
    extern __shared__ __align__(1024) unsigned char score_smem_raw[];
    // swizzled TMA tiles must start on a 1024-byte boundary
    unsigned char* score_smem = score_smem_raw + ((1024 - (smem_u32(score_smem_raw) & 1023)) & 1023);
    const int lane = threadIdx.x & 31, wl = threadIdx.x >> 5, grp = lane >> 2, tq = lane & 3;
    const uint32_t tiles = smem_u32(score_smem) + wl * S * TB;
    const uint32_t bars = smem_u32(score_smem) + kScoreWarps * S * TB + wl * S * 8;
    int4* table = reinterpret_cast<int4*>(score_smem + kScoreWarps * S * (TB + 8)) + wl * 64;
    int* smem_cum = reinterpret_cast<int*>(score_smem + kScoreWarps * S * (TB + 8) + kScoreWarps * 64 * 16);
    __shared__ int warp_tot[kScoreWarps];
    const int total = units_prefix(a.ctx_lens, a.B, P, a.max_blocks, a.Hkv, smem_cum, warp_tot);
    const int gwarp = blockIdx.x * kScoreWarps + wl;
    const int nwarps = gridDim.x * kScoreWarps;
    const int share = (total + nwarps - 1) / nwarps;
    const int u0 = gwarp * share;
    const int u1 = min(u0 + share, total);
    if (u0 >= u1) return;
    const int ntiles = (u1 - u0) * kTiles;

    if (lane == 0) {
        for (int st = 0; st < S; ++st) mbar_init(bars + 8 * st, 1);
        fence_mbar_init();
    }
    __syncwarp();

    // units [u0 + 32k, u0 + 32k + 32) -> table slot k & 1, one lane per unit:
    // (sequence, kv head, block, page or -1)
    auto resolve = [&](int k) {
        const int u = u0 + 32 * k + lane;
        int4 e = make_int4(0, 0, 0, -1);
        if (u < u1) {
            int lo = 0, hi = a.B - 1;   // largest b with cum[b] <= u
            while (lo < hi) {
                const int mid = (lo + hi + 1) >> 1;
                if (smem_cum[mid] <= u) lo = mid; else hi = mid - 1;
            }
            const int nb = seq_blocks(__ldg(a.ctx_lens + lo), P, a.max_blocks);
            const int r = u - smem_cum[lo];
            e.x = lo;
            e.y = r / nb;
            e.z = r - e.y * nb;
            const int pg = __ldg(a.block_table + (long long)lo * a.max_blocks + e.z);
            e.w = (pg >= 0 && (long long)pg < a.num_pages) ? pg : -1;
        }
        table[(k & 1) * 32 + lane] = e;
        __syncwarp();
    };
    auto entry = [&](int item) -> int4 {
        const int r = item - u0;
        return table[((r >> 5) & 1) * 32 + (r & 31)];
    };
    // issue the TMA copies of tile i into stage st (one elected lane)
    auto issue = [&](int i, int st) {
        if (lane == 0) {
            const int item = u0 + i / kTiles;
            const int tile = i - (i / kTiles) * kTiles;
            const int4 e = entry(item);
            const uint32_t bar = bars + 8 * st;
            if (e.w >= 0) {
                mbar_arrive_expect_tx(bar, TB);
                const int y = (e.w * a.Hkv + e.y) * P + tile * 16;
#pragma unroll
                for (int h = 0; h < H; ++h) tma_load_2d(tiles + st * TB + h * 2048, &kmap, 64 * h, y, bar);
            } else {
                mbar_arrive(bar);   // nothing to copy: the block's page id is invalid
            }
        }
    };

    resolve(0);
    if (ntiles > 32 * kTiles) resolve(1);
#pragma unroll 1
    for (int st = 0; st < S && st < ntiles; ++st) issue(st, st);

    uint4 qf[H][2];
    int q_b = -1, q_kvh = -1;
    float xs[kTiles][4];
    float ss[kTiles][2];          // stored surprisal of token slots grp, grp + 8
    int i = 0;
    bool timed_out = false;
#pragma unroll 1
    for (; i < ntiles; ++i) {
        const int st = i % S;
        const int item = u0 + i / kTiles;
        const int tile = i - (i / kTiles) * kTiles;
        if (tile == 0 && ((item - u0) & 31) == 0 && item > u0 && item - u0 + 32 < u1 - u0)
            resolve(((item - u0) >> 5) + 1);
        if (!mbar_wait(bars + 8 * st, (uint32_t)((i / S) & 1), a.wait_iters)) {
            timed_out = true;
            break;
        }
        const int4 e = entry(item);
        const int b = e.x, kvh = e.y, blk = e.z;
        if (b != q_b || kvh != q_kvh) {
            q_b = b;
            q_kvh = kvh;
            const int h = kvh * a.g + grp;
#pragma unroll
            for (int hh = 0; hh < H; ++hh)
#pragma unroll
                for (int c = 0; c < 2; ++c)
                    qf[hh][c] = grp < a.g ? __ldg(reinterpret_cast<const uint4*>(
                                                a.q + ((long long)b * a.Hq + h) * D + 64 * hh + 16 * tq + 8 * c))
                                          : make_uint4(0, 0, 0, 0);
        }
        // q.k on the tensor cores: tokens = M, heads = N, head_dim = K; the
        // thread's 16-byte chunks (2tq + c of each 64-element half) are read
        // conflict-free from the swizzled tile, the same d permutation is used
        // in the query fragment
        const uint32_t tb = tiles + st * TB;
        float acc[4] = {0.f, 0.f, 0.f, 0.f}, acc2[4] = {0.f, 0.f, 0.f, 0.f};   // two MMA chains
#pragma unroll
        for (int hh = 0; hh < H; ++hh)
#pragma unroll
            for (int c = 0; c < 2; ++c) {
                const uint4 lo = lds_u4(tb + hh * 2048 + swz128(grp, 2 * tq + c));
                const uint4 hi = lds_u4(tb + hh * 2048 + swz128(grp + 8, 2 * tq + c));
                mma_bf16_16x8x16(acc, lo.x, hi.x, lo.y, hi.y, qf[hh][c].x, qf[hh][c].y);
                mma_bf16_16x8x16(acc2, lo.z, hi.z, lo.w, hi.w, qf[hh][c].z, qf[hh][c].w);
            }
#pragma unroll
        for (int e2 = 0; e2 < 4; ++e2) acc[e2] += acc2[e2];
        // the tile's shared memory may be refilled now
        __syncwarp();
        fence_proxy_async();
        if (i + S < ntiles) issue(i + S, st);

        // token slots grp, grp+8 of this tile; heads 2tq, 2tq+1
        const int L = __ldg(a.ctx_lens + b);
        const int valid_tok = min(P, L - blk * P) - tile * 16;
        const bool ok = e.w >= 0;
        float x4[4];
        x4[0] = (ok && grp < valid_tok) ? acc[0] * a.scale : -kInf;
        x4[1] = (ok && grp < valid_tok) ? acc[1] * a.scale : -kInf;
        x4[2] = (ok && grp + 8 < valid_tok) ? acc[2] * a.scale : -kInf;
        x4[3] = (ok && grp + 8 < valid_tok) ? acc[3] * a.scale : -kInf;
#pragma unroll
        for (int tt = 0; tt < kTiles; ++tt)      // static indices keep xs in registers
            if (tt == tile)
#pragma unroll
                for (int ee = 0; ee < 4; ++ee) xs[tt][ee] = x4[ee];
        if (a.tok_surp) {
            // score mode E: the surprisal of each token, paged like the keys
            const float* sp = a.tok_surp + (long long)e.w * P + tile * 16 + grp;
            const float s0 = (ok && grp < valid_tok) ? __ldg(sp) : 0.f;
            const float s1 = (ok && grp + 8 < valid_tok) ? __ldg(sp + 8) : 0.f;
#pragma unroll
            for (int tt = 0; tt < kTiles; ++tt)
                if (tt == tile) { ss[tt][0] = s0; ss[tt][1] = s1; }
        }
        const long long unit = ((long long)b * a.Hkv + kvh) * a.max_blocks + blk;
        if (a.token_scores) {
            float* ts = a.token_scores + (unit * P + tile * 16) * a.g;
            const int h0 = 2 * tq, h1 = 2 * tq + 1;
            if (h1 < a.g && (a.g & 1) == 0) {
                *reinterpret_cast<float2*>(ts + grp * a.g + h0) = make_float2(x4[0], x4[1]);
                *reinterpret_cast<float2*>(ts + (grp + 8) * a.g + h0) = make_float2(x4[2], x4[3]);
            } else {
                if (h0 < a.g) {
                    ts[grp * a.g + h0] = x4[0];
                    ts[(grp + 8) * a.g + h0] = x4[2];
                }
                if (h1 < a.g) {
                    ts[grp * a.g + h1] = x4[1];
                    ts[(grp + 8) * a.g + h1] = x4[3];
                }
            }
        }
        if (tile == kTiles - 1) {
            // block stats for heads 2tq (j = 0) and 2tq + 1 (j = 1)
#pragma unroll
            for (int j = 0; j < 2; ++j) {
                float m = -kInf;
#pragma unroll
                for (int tt = 0; tt < kTiles; ++tt) m = fmaxf(m, fmaxf(xs[tt][j], xs[tt][j + 2]));
                m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 4));
                m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 8));
                m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 16));
                // l1 = (sum e^{x-m}) - 1, kept exact: the tokens below the max are
                // summed and every further token AT the max adds exactly 1, so a
                // block dominated by one token keeps its small remainder.
                float l1 = 0.f, u = 0.f, neq = 0.f, es = 0.f;
                if (m != -kInf) {
#pragma unroll
                    for (int tt = 0; tt < kTiles; ++tt) {
#pragma unroll
                        for (int ee = 0; ee < 2; ++ee) {
                            const float d = xs[tt][j + 2 * ee] - m;
                            const float w = fast_ex2(d * kLog2e);
                            l1 += d < 0.f ? w : 0.f;
                            neq += d == 0.f ? 1.f : 0.f;
                            u = fmaf(w, fmaxf(d, -1e30f), u);
                            if (a.tok_surp) es = fmaf(w, ss[tt][ee], es);
                        }
                    }
                }
#pragma unroll
                for (int o = 4; o <= 16; o <<= 1) {
                    l1 += __shfl_xor_sync(0xffffffffu, l1, o);
                    u += __shfl_xor_sync(0xffffffffu, u, o);
                    neq += __shfl_xor_sync(0xffffffffu, neq, o);
                    if (a.tok_surp) es += __shfl_xor_sync(0xffffffffu, es, o);
                }
                l1 += neq - 1.f;
                const int h = 2 * tq + j;
                if (grp == 0 && h < a.g) a.stats[unit * a.g + h] = make_float4(m, l1, u, es);
            }
        }
    }
    if (timed_out) {
        // a copy never arrived: let the copies still in flight land (bounded
        // by the default limit), then mark every block this warp did not
        // finish with NaN stats, which the keep-set pass reports as
        // ETI_ERRF_TIMEOUT for its sequence; l - 1 = +inf instead of NaN also
        // says that a copy was still in flight when the drain gave up
        // (ETI_ERRF_DRAIN)
        bool drained = true;
        for (int k = i; k < ntiles && k < i + S; ++k)
            drained &= mbar_wait(bars + 8 * (k % S), (uint32_t)((k / S) & 1), kMaxWaitIters);
        const float nan = __int_as_float(0x7fc00000);
        const float l1_mark = drained ? nan : kInf;
        for (int item = u0 + i / kTiles; item < u1; ++item) {
            if (((item - u0) & 31) == 0 && item > u0) resolve((item - u0) >> 5);
            const int4 e = entry(item);
            const long long unit = ((long long)e.x * a.Hkv + e.y) * a.max_blocks + e.z;
            if (lane < a.g) a.stats[unit * a.g + lane] = make_float4(nan, l1_mark, nan, 0.f);
        }
    }
}

// ---------------------------------------------------------------------------
// Zeroes the per-sequence error words before the keep-set kernel ORs its bits
// in (every kv head of a sequence adds its own).  A kernel, not a memset: a
// memset node in a captured CUDA graph cost about 30 us per replay here, and
// after a kernel the keep-set kernel keeps its programmatic launch overlap.
__global__ void __launch_bounds__(256) clear_words_kernel(uint32_t* w, int n) {
    pdl_trigger();
    pdl_wait();
    for (int i = blockIdx.x * 256 + threadIdx.x; i < n; i += gridDim.x * 256) w[i] = 0u;
}

}  // namespace eti

using namespace eti;

int eti_launch_score_blocks(const uint16_t* q, const uint16_t* k_cache, const int32_t* block_table,
                            const int32_t* ctx_lens, int B, int Hq, int Hkv, int D, int P,
                            int max_blocks, long long num_pages, float scale, const float* tok_surp,
                            float* token_scores, float4* stats, cudaStream_t stream) {
    if (B == 0) return ETI_OK;
    if (num_pages <= 0) {
        // no page can be valid: every sequence with blocks is reported by the
        // keep-set pass; nothing to score
        return ETI_OK;
    }
    ScoreArgs a;
    a.q = q; a.k_cache = k_cache; a.block_table = block_table; a.ctx_lens = ctx_lens;
    a.B = B; a.Hq = Hq; a.Hkv = Hkv; a.g = Hq / Hkv; a.max_blocks = max_blocks;
    a.num_pages = num_pages; a.scale = scale; a.token_scores = token_scores; a.stats = stats;
    a.tok_surp = tok_surp;
    a.wait_iters = eti_wait_limit();
    // tile row coordinates are int32 on the device
    if (num_pages * Hkv * P >= (1LL << 31)) return ETI_ERR_UNSUPPORTED;
    CUtensorMap kmap;
    int st = eti_make_kv_tensor_map(&kmap, k_cache, num_pages * Hkv * P, D);
    if (st != ETI_OK) return st;
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    cudaError_t e;
#define ETI_SCORE_CASE(DD, PP)                                                              \
    if (D == DD && P == PP) {                                                               \
        auto k = score_blocks_kernel<DD, PP>;                                               \
        const size_t smem = score_smem_bytes<DD, PP>(B);                                    \
        const int grid = (smem + 2048 <= 233472 / 2 ? 2 : 1) * sms;   /* CTAs that fit */   \
        cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);    \
        e = eti_launch_pdl(k, dim3(grid), dim3(kScoreThreads), smem, stream, kmap, a);      \
        return e == cudaSuccess ? ETI_OK : ETI_ERR_CUDA;                                    \
    }
    ETI_SCORE_CASE(128, 16)
    ETI_SCORE_CASE(128, 32)
    ETI_SCORE_CASE(64, 16)
    ETI_SCORE_CASE(64, 32)
#undef ETI_SCORE_CASE
    return ETI_ERR_UNSUPPORTED;
}

cudaError_t eti_launch_prune_wide(const eti::FinArgs& a, int segs, int sms, cudaStream_t stream);
bool eti_prune_tile_fits(int max_blocks, int g, int B_min, int segs, int sms);
cudaError_t eti_launch_prune_tile(const eti::FinArgs& a, cudaStream_t stream);

int eti_launch_prune_finalize(const float4* stats, const int32_t* ctx_lens, const int32_t* block_table,
                              long long num_pages, int B, int Hq, int Hkv, int P, int max_blocks,
                              const float* theta, int B_min, int score_mode, int given,
                              const uint8_t* given_mask,
                              const int32_t* given_idx, const int32_t* given_cnt, uint8_t* keep_mask,
                              int32_t* kept_idx, int32_t* kept_cnt, float* block_score,
                              float* kept_norm, uint32_t* err, cudaStream_t stream) {
    if (B == 0) return ETI_OK;
    FinArgs a;
    a.stats = stats; a.ctx_lens = ctx_lens; a.block_table = block_table; a.num_pages = num_pages;
    a.B = B; a.Hq = Hq; a.Hkv = Hkv; a.g = Hq / Hkv; a.P = P; a.max_blocks = max_blocks;
    a.theta = theta; a.B_min = B_min; a.score_mode = score_mode; a.given = given; a.given_mask = given_mask;
    a.given_idx = given_idx; a.given_cnt = given_cnt; a.keep_mask = keep_mask;
    a.kept_idx = kept_idx; a.kept_cnt = kept_cnt; a.block_score = block_score;
    a.kept_norm = kept_norm; a.err = err;
    a.share_cache = 0;
    const int grid = B * Hkv;
    cudaError_t e = cudaSuccess;
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (err) {
        // programmatic launch: it waits for the kernel before it inside
        // (griddepcontrol.wait), and the keep-set kernel overlaps its own
        // launch with it
        if (eti_launch_pdl(clear_words_kernel, dim3((B + 255) / 256), dim3(256), 0, stream, err, B) != cudaSuccess)
            return ETI_ERR_CUDA;
    }
    // the rule mode with segments of up to 8192 block-heads, or up to 32768
    // with B_min <= 1 and few segments (a cluster of CTAs a segment): the
    // tile kernel (the stats staged in shared memory, work that follows each
    // segment's length); the rest, and a cluster launch the device refuses:
    // prune_wide.cu
    if (!given && theta && eti_prune_tile_fits(max_blocks, a.g, B_min, grid, sms)) {
        e = eti_launch_prune_tile(a, stream);
        if (e != cudaSuccess && (long long)max_blocks * a.g > 8192) {
            (void)cudaGetLastError();
            e = eti_launch_prune_wide(a, grid, sms, stream);
        }
    } else {
        e = eti_launch_prune_wide(a, grid, sms, stream);
    }
    return e == cudaSuccess ? ETI_OK : ETI_ERR_CUDA;
}
