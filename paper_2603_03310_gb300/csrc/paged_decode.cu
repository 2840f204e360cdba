// paged_decode.cu -- GQA paged decode attention restricted to the kept blocks
// (Section 3.2: attention is computed over B_t only, renormalised over the
// kept tokens).
//
// The scorer already produced x_i = scale q_h . k_i for every token and the
// finalizer the kept-token softmax normaliser (M_h, l_h) of every query head,
// so this pass reads only the kept V pages and their scores:
//   out_h = (1 / l_h) sum_{i kept} e^{x_i - M_h} v_i .
// The weights are normalised against a fixed M_h, so partial sums over
// different block ranges simply add (no rescaling).
//
// Work split (warp-level stream-K): the kept blocks of all (sequence, kv head)
// segments form one list; warp w takes the contiguous range
// [w*share, (w+1)*share).  Each warp streams its 16-token tiles through a
// private ring of shared-memory stages filled by the Tensor Memory
// Accelerator: one elected lane issues two 2-D tiled copies (64-element boxes
// with the 128-byte swizzle, so the fragment reads below are conflict-free)
// and a 1-D bulk copy of the tile's scores per stage, completing on the
// stage's mbarrier; every wait is bounded.  Page ids are resolved 32 blocks at
// a time, one lane per block, into a small table a batch ahead of use.  p.V
// runs on bf16 m16n8k16 tensor-core tiles (head_dim = M, query heads = N,
// tokens = K): each A fragment (V^T, 16 x 16) is one ldmatrix.x4.trans from
// the swizzled stage, the probabilities form the B fragment.
// A segment that lies inside one warp's range is written straight to `out`;
// otherwise the warp's part goes to partial slot (warp + segment), and the
// warp that closes the segment's ticket last adds its slots in warp order
// (deterministic) and writes the output: no second kernel, no waiting.
//
// The plan kernel that runs first forms the prefix of kept counts, each
// warp's first segment, zeroes the tickets, and writes every sequence's error
// word (context length and page ids checked once, one warp per sequence).
#include <cstring>

#include "common.cuh"

namespace eti {

constexpr int kDecWarps = 8;
constexpr int kDecThreads = kDecWarps * 32;
constexpr int kPlanThreads = 1024;
constexpr int kPlanSmemSeg = 4096;   // segments whose prefix the plan keeps in shared memory

// --------------------------------------------------------------------------
// plan: prefix of kept counts, the per-warp share, each warp's first
// segment, zeroed tickets (CTA 0); the error word of every sequence (the
// other CTAs, one warp per sequence)
struct PlanArgs {
    const int32_t* kept_cnt;
    const int32_t* ctx_lens;
    const int32_t* block_table;
    long long num_pages;
    int B, Hkv, P;
    int nseg, nwarps, max_blocks;
    int* cum;       // [nseg + 1]
    int* info;      // [0] = total kept blocks, [1] = share per warp
    int* warp_seg;  // [nwarps]
    int* ticket;    // [nseg]
    uint32_t* err;  // [B]
};

__global__ void __launch_bounds__(kPlanThreads) decode_plan_kernel(const PlanArgs a) {
    pdl_trigger();
    pdl_wait();
    const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
    if (blockIdx.x > 0) {
        const int b = (blockIdx.x - 1) * (kPlanThreads / 32) + w;
        if (b >= a.B) return;
        const int L = a.ctx_lens[b];
        const bool bad_ctx = L < 0 || L > a.max_blocks * a.P;
        const int nb = bad_ctx ? 0 : (L + a.P - 1) / a.P;
        const bool bad = __any_sync(0xffffffffu, any_bad_page(a.block_table + (long long)b * a.max_blocks,
                                                              lane, 32, nb, a.num_pages));
        if (lane == 0) a.err[b] = bad_ctx ? ETI_ERRF_BAD_CTX : (bad ? ETI_ERRF_BAD_PAGE : 0u);
        return;
    }
    __shared__ int wsum[kPlanThreads / 32];
    __shared__ int scum[kPlanSmemSeg + 1];   // cum[0 .. kPlanSmemSeg], kept for the second loop
    int carry = 0;
    for (int base = 0; base < a.nseg; base += kPlanThreads) {
        const int s = base + tid;
        const int v = s < a.nseg ? min(max(a.kept_cnt[s], 0), a.max_blocks) : 0;
        int x = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x += y;
        }
        if (lane == 31) wsum[w] = x;
        __syncthreads();
        int ofs = 0, tot = 0;
        for (int i = 0; i < kPlanThreads / 32; ++i) {
            if (i < w) ofs += wsum[i];
            tot += wsum[i];
        }
        if (s < a.nseg) {
            a.cum[s] = carry + ofs + x - v;
            a.ticket[s] = 0;
            if (s <= kPlanSmemSeg) scum[s] = carry + ofs + x - v;
        }
        carry += tot;
        __syncthreads();
    }
    const int total = carry;
    // at least 4 kept blocks per warp (a small batch spreads over more warps:
    // on 4 sequences of 64 to 256 tokens the call took 32.8 us with at least
    // 32 a warp, 22.5 with 16, 18.4 with 8, 14.4 with 4; the large workloads'
    // shares are far above the floor)
    const int share = max(4, (total + a.nwarps - 1) / a.nwarps);
    if (tid == 0) {
        if (a.nseg <= kPlanSmemSeg) scum[a.nseg] = total;
        a.cum[a.nseg] = total;
        a.info[0] = total;
        a.info[1] = share;
    }
    for (int c = tid; c < a.nwarps; c += kPlanThreads) a.warp_seg[c] = a.nseg;
    __syncthreads();
    for (int s = tid; s < a.nseg; s += kPlanThreads) {
        const int lo = s + 1 <= kPlanSmemSeg ? scum[s] : a.cum[s];
        const int hi = s + 1 <= kPlanSmemSeg ? scum[s + 1] : a.cum[s + 1];
        if (hi <= lo) continue;
        const int c0 = (lo + share - 1) / share, c1 = min((hi + share - 1) / share, a.nwarps);
        for (int c = c0; c < c1; ++c) a.warp_seg[c] = s;
    }
}

// --------------------------------------------------------------------------
struct DecArgs {
    const uint16_t* v_cache;
    const int32_t* block_table;
    const int32_t* ctx_lens;
    const int32_t* kept_idx;       // [nseg][max_blocks]
    const float* token_scores;     // [nseg][max_blocks][P][g]
    const float* kept_norm;        // [B][Hq][2]
    const int* cum;
    const int* info;
    const int* warp_seg;
    int B, Hq, Hkv, g, max_blocks;
    long long num_pages;
    uint16_t* out;                 // bf16 [B][Hq][D]
    float* partial;                // [(nwarps + nseg)][g][D]
    int* ticket;                   // [nseg], zeroed by the plan kernel
    uint32_t* err;                 // [B], written by the plan kernel
    int wait_iters;                // polls before a tile wait gives up (eti_set_wait_limit)
};

template <int D>
struct DecLayout {
    static constexpr int kTile = 16 * D * 2;      // bytes of one 16-token V tile
    static constexpr int kStages = D == 128 ? 3 : 5;
};

// bytes of one tile's scores (16 tokens x g heads, fp32)
__host__ __device__ inline int dec_score_bytes(int g) { return 16 * g * 4; }

template <int D>
__host__ __device__ inline size_t dec_smem_bytes(int g) {
    return 1024 + (size_t)kDecWarps * DecLayout<D>::kStages * (DecLayout<D>::kTile + dec_score_bytes(g) + 8)
           + (size_t)kDecWarps * 64 * 16;
}

// A-fragment rows owned by a thread (tq = lane & 3): 2tq, 2tq+1, 2tq+8, 2tq+9
__device__ __forceinline__ int frag_row(int tq, int k) { return 2 * tq + (k & 1) + (k >> 1) * 8; }

template <int D, int P>
__global__ void __launch_bounds__(kDecThreads, 2)
paged_decode_kernel(const __grid_constant__ CUtensorMap vmap, const DecArgs a) {
    constexpr int kTiles = P / 16;
    constexpr int J = D / 16;                    // MMAs per 16-token tile
    constexpr int S = DecLayout<D>::kStages;
    constexpr int TB = DecLayout<D>::kTile;
    constexpr int H = D / 64;                    // 64-element boxes per tile row
    pdl_trigger();
    pdl_wait();
    const int SB = dec_score_bytes(a.g);
    extern __shared__ __align__(1024) unsigned char dec_smem_raw[];
    unsigned char* dec_smem = dec_smem_raw + ((1024 - (smem_u32(dec_smem_raw) & 1023)) & 1023);
    const int lane = threadIdx.x & 31, wl = threadIdx.x >> 5, grp = lane >> 2, tq = lane & 3;
    const int warp = blockIdx.x * kDecWarps + wl;
    const int total = a.info[0], share = a.info[1];
    const int u0 = warp * share;
    const int u1 = min(u0 + share, total);
    const int nseg = a.B * a.Hkv;
    // segments with nothing kept have no writer: their output is zeroed here
    auto zero_empty = [&]() {
        for (int s = warp; s < nseg; s += gridDim.x * kDecWarps) {
            if (__ldg(a.cum + s + 1) > __ldg(a.cum + s)) continue;
            const int b = s / a.Hkv, kvh = s - b * a.Hkv;
            uint16_t* o = a.out + ((long long)b * a.Hq + kvh * a.g) * D;
            for (int e = lane * 8; e < a.g * D; e += 256) *reinterpret_cast<uint4*>(o + e) = make_uint4(0, 0, 0, 0);
        }
    };
    if (u0 >= u1) {
        zero_empty();
        return;
    }
    const int ntiles = (u1 - u0) * kTiles;
    const uint32_t tiles = smem_u32(dec_smem) + wl * S * TB;
    const uint32_t scores = smem_u32(dec_smem) + kDecWarps * S * TB + wl * S * SB;
    const uint32_t bars = smem_u32(dec_smem) + kDecWarps * S * (TB + SB) + wl * S * 8;
    int4* table = reinterpret_cast<int4*>(dec_smem + kDecWarps * S * (TB + SB + 8)) + wl * 64;
    const int sbytes = SB;                       // one tile's scores (a multiple of 16)

    if (lane == 0) {
        for (int st = 0; st < S; ++st) mbar_init(bars + 8 * st, 1);
        fence_mbar_init();
    }
    __syncwarp();

    // items [u0 + 32k, u0 + 32k + 32) -> table slot k & 1: (segment, block,
    // page or -1, valid tokens of the block)
    int seg_hint = a.warp_seg[warp];
    auto resolve = [&](int k) {
        const int u = u0 + 32 * k + lane;
        int4 e = make_int4(seg_hint, 0, -1, 0);
        if (u < u1) {
            int s = seg_hint;
            while (s < nseg - 1 && __ldg(a.cum + s + 1) <= u) ++s;
            e.x = s;
            const int b = s / a.Hkv;
            const int L = __ldg(a.ctx_lens + b);
            const int nb = seq_blocks(L, P, a.max_blocks);
            const int blk = __ldg(a.kept_idx + (long long)s * a.max_blocks + (u - __ldg(a.cum + s)));
            if (blk >= 0 && blk < nb) {
                const int pg = __ldg(a.block_table + (long long)b * a.max_blocks + blk);
                if (pg >= 0 && (long long)pg < a.num_pages) {
                    e.y = blk;
                    e.z = pg;
                    e.w = min(P, L - blk * P);
                }
            }
        }
        table[(k & 1) * 32 + lane] = e;
        seg_hint = __shfl_sync(0xffffffffu, e.x, 31);
        __syncwarp();
    };
    auto entry = [&](int item) -> int4 {
        const int r = item - u0;
        return table[((r >> 5) & 1) * 32 + (r & 31)];
    };
    auto issue = [&](int i, int st) {
        if (lane == 0) {
            const int item = u0 + i / kTiles;
            const int tile = i - (i / kTiles) * kTiles;
            const int4 e = entry(item);
            const uint32_t bar = bars + 8 * st;
            if (e.z >= 0) {
                const int kvh = e.x - (e.x / a.Hkv) * a.Hkv;
                mbar_arrive_expect_tx(bar, TB + sbytes);
                const int y = (e.z * a.Hkv + kvh) * P + tile * 16;
#pragma unroll
                for (int h = 0; h < H; ++h) tma_load_2d(tiles + st * TB + h * 2048, &vmap, 64 * h, y, bar);
                bulk_load_1d(scores + st * SB,
                             a.token_scores + (((long long)e.x * a.max_blocks + e.y) * P + tile * 16) * a.g,
                             sbytes, bar);
            } else {
                mbar_arrive(bar);
            }
        }
    };

    float acc[J][4];
#pragma unroll
    for (int j = 0; j < J; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;

    // the last warp of a split segment: add the slots (warp + seg) of warps
    // w0..w1 in warp order, normalise, write bf16 (zeros for a bad sequence)
    auto merge = [&](int seg, int lo, int hi, bool bad) {
        const int b = seg / a.Hkv, kvh = seg - b * a.Hkv;
        const int w0 = lo / share, nw = (hi - 1) / share - w0 + 1;
        const long long stride = (long long)a.g * D;      // floats between consecutive slots
        const float4* base = reinterpret_cast<const float4*>(a.partial + (long long)(w0 + seg) * stride);
        const int n4 = a.g * D / 4;                         // float4 per slot
        constexpr int kM = D / 16;                          // float4 per lane for g = 8
        float4 v[kM];
#pragma unroll
        for (int k = 0; k < kM; ++k) v[k] = make_float4(0.f, 0.f, 0.f, 0.f);
        // four slots' loads in flight at a time (the sums wait on L2 latency)
#pragma unroll 4
        for (int w = 0; w < nw; ++w) {
#pragma unroll
            for (int k = 0; k < kM; ++k) {
                const int e4 = lane + 32 * k;
                if (e4 < n4) {
                    // L2 reads: the other warps' slots were published by their tickets
                    const float4 x = __ldcg(base + (long long)w * (stride / 4) + e4);
                    v[k].x += x.x; v[k].y += x.y; v[k].z += x.z; v[k].w += x.w;
                }
            }
        }
#pragma unroll
        for (int k = 0; k < kM; ++k) {
            const int e4 = lane + 32 * k;
            if (e4 < n4) {
                const int h = (4 * e4) / D, d = 4 * e4 - h * D;
                const float l = __ldg(a.kept_norm + ((long long)b * a.Hq + kvh * a.g + h) * 2 + 1);
                const float inv = (!bad && l > 0.f) ? 1.f / l : 0.f;
                *reinterpret_cast<uint2*>(a.out + ((long long)b * a.Hq + kvh * a.g + h) * D + d) =
                    make_uint2(pack_bf16x2(v[k].x * inv, v[k].y * inv), pack_bf16x2(v[k].z * inv, v[k].w * inv));
            }
        }
    };

    // write the accumulated segment: straight to `out` when the whole segment
    // is in this warp's range, else into partial slot (warp + seg) and take a
    // ticket; the warp that takes the segment's last ticket merges the slots
    auto flush = [&](int seg) {
        const int b = seg / a.Hkv, kvh = seg - b * a.Hkv;
        const int lo = __ldg(a.cum + seg), hi = __ldg(a.cum + seg + 1);
        const bool whole = lo >= u0 && hi <= u1;
        const bool bad = (a.err[b] & (ETI_ERRF_BAD_CTX | ETI_ERRF_BAD_PAGE)) != 0u;
        // acc[j][e], acc[j][2 + e]: head 2 tq + e at d = 16 j + grp and 16 j + 8 + grp
#pragma unroll
        for (int e = 0; e < 2; ++e) {
            const int h = 2 * tq + e;
            if (h < a.g) {
                if (whole) {
                    const float l = __ldg(a.kept_norm + ((long long)b * a.Hq + kvh * a.g + h) * 2 + 1);
                    const float inv = (!bad && l > 0.f) ? 1.f / l : 0.f;
                    uint16_t* o = a.out + ((long long)b * a.Hq + kvh * a.g + h) * D + grp;
#pragma unroll
                    for (int j = 0; j < J; ++j) {
                        o[16 * j] = __bfloat16_as_ushort(__float2bfloat16_rn(acc[j][e] * inv));
                        o[16 * j + 8] = __bfloat16_as_ushort(__float2bfloat16_rn(acc[j][2 + e] * inv));
                    }
                } else {
                    float* o = a.partial + ((long long)(warp + seg) * a.g + h) * D + grp;
#pragma unroll
                    for (int j = 0; j < J; ++j) {
                        o[16 * j] = acc[j][e];
                        o[16 * j + 8] = acc[j][2 + e];
                    }
                }
            }
        }
#pragma unroll
        for (int j = 0; j < J; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;
        if (!whole) {
            __threadfence();          // this lane's part of the slot, before the ticket
            __syncwarp();
            int last = 0;
            if (lane == 0) last = atomicAdd(a.ticket + seg, 1) == (hi - 1) / share - lo / share;
            if (__shfl_sync(0xffffffffu, last, 0)) {
                __threadfence();
                merge(seg, lo, hi, bad);
            }
        }
    };

    resolve(0);
    if (u1 - u0 > 32) resolve(1);
#pragma unroll 1
    for (int st = 0; st < S && st < ntiles; ++st) issue(st, st);

    int cur_seg = -1;
    float Mh = 0.f;
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
        if (e.x != cur_seg) {
            if (cur_seg >= 0) flush(cur_seg);
            cur_seg = e.x;
            const int b = cur_seg / a.Hkv, kvh = cur_seg - b * a.Hkv;
            Mh = grp < a.g ? __ldg(a.kept_norm + ((long long)b * a.Hq + kvh * a.g + grp) * 2) : 0.f;
        }
        const uint32_t tb = tiles + st * TB, sc = scores + st * SB;
        // valid rows of this tile, in [0, 16] (the second tile of a 32-token page
        // can lie wholly past the sequence end)
        const int vrow = e.z >= 0 ? max(0, min(16, e.w - tile * 16)) : 0;
        if (vrow < 16) {
            // rows past the sequence end (or of a skipped page) hold whatever the
            // stage holds: zero them, so that a finite weight meets a zero row
            for (int c = lane; c < (16 - vrow) * (D / 8); c += 32) {
                const int row = vrow + c / (D / 8), ch = c % (D / 8);
                sts_zero_u4(tb + (ch >> 3) * 2048 + row * 128 + (ch & 7) * 16);
            }
            __syncwarp();
        }
        float p[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int row = frag_row(tq, k);
            const float x = (row < vrow && grp < a.g) ? lds_f32(sc + (row * a.g + grp) * 4) : 0.f;
            // kept tokens have x <= M_h; zeroed rows get a finite weight against a zero row
            p[k] = fast_ex2(fminf((x - Mh) * kLog2e, 0.f));
        }
        // A fragments of V^T (head_dim = M, tokens = K), MMA j on d = 16 j .. 16 j + 15:
        // matrix q of lane l is (tokens 8 (q >> 1) .. +7, d = 16 j + 8 (q & 1) .. +7)
        uint32_t af[J][4];
        {
            const int q = lane >> 3, rr = (lane & 7) + (q >> 1) * 8;
#pragma unroll
            for (int j = 0; j < J; ++j) {
                const int d = 16 * j + 8 * (q & 1);
                ldsm_x4_trans(af[j], tb + (d >> 6) * 2048 + swz128(rr, (d & 63) >> 3));
            }
        }
        // the stage may be refilled now
        __syncwarp();
        fence_proxy_async();
        if (i + S < ntiles) issue(i + S, st);
        const uint32_t b0 = pack_bf16x2(p[0], p[1]);
        const uint32_t b1 = pack_bf16x2(p[2], p[3]);
#pragma unroll
        for (int j = 0; j < J; ++j) mma_bf16_16x8x16(acc[j], af[j][0], af[j][1], af[j][2], af[j][3], b0, b1);
    }
    if (timed_out) {
        // a copy never arrived: let the ones in flight land (bounded), flag
        // every sequence of the rest of this range, and still close their
        // segments (tickets included) so no output is left unwritten
        // (the drain waits with the default limit; a copy still in flight
        // after it is reported as ETI_ERRF_DRAIN)
        bool drained = true;
        for (int k = i; k < ntiles && k < i + S; ++k)
            drained &= mbar_wait(bars + 8 * (k % S), (uint32_t)((k / S) & 1), kMaxWaitIters);
        const uint32_t bits = ETI_ERRF_TIMEOUT | (drained ? 0u : ETI_ERRF_DRAIN);
        for (int sg = cur_seg >= 0 ? cur_seg : a.warp_seg[warp]; sg < nseg && __ldg(a.cum + sg) < u1; ++sg) {
            if (__ldg(a.cum + sg + 1) <= __ldg(a.cum + sg)) continue;
            if (lane == 0) atomicOr(a.err + sg / a.Hkv, bits);
            flush(sg);
        }
        zero_empty();
        return;
    }
    if (cur_seg >= 0) flush(cur_seg);
    zero_empty();
}

// CTAs of the decode kernel per SM for this shape (as many as fit, up to 2)
inline int dec_ctas_per_sm(int D, int g) {
    const size_t sm = D == 128 ? dec_smem_bytes<128>(g) : dec_smem_bytes<64>(g);
    return sm + 1024 <= 233472 / 2 ? 2 : 1;
}

}  // namespace eti

using namespace eti;

// warps of the persistent decode grid on the current device
int eti_decode_nwarps(int D, int g) {
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    return dec_ctas_per_sm(D, g) * sms * kDecWarps;
}

int eti_launch_decode(const uint16_t* v_cache, const int32_t* block_table, const int32_t* ctx_lens,
                      const int32_t* kept_idx, const int32_t* kept_cnt, const float* token_scores,
                      const float* kept_norm, int B, int Hq, int Hkv, int D, int P, int max_blocks,
                      long long num_pages, uint16_t* out, uint32_t* err, int* plan_cum,
                      int* plan_info, int* plan_warp_seg, int* plan_ticket, float* partial,
                      int nwarps, cudaStream_t stream) {
    if (B == 0) return ETI_OK;
    const int nseg = B * Hkv;
    PlanArgs pa;
    pa.kept_cnt = kept_cnt; pa.ctx_lens = ctx_lens; pa.block_table = block_table;
    pa.num_pages = num_pages; pa.B = B; pa.Hkv = Hkv; pa.P = P;
    pa.nseg = nseg; pa.nwarps = nwarps; pa.max_blocks = max_blocks;
    pa.cum = plan_cum; pa.info = plan_info; pa.warp_seg = plan_warp_seg;
    pa.ticket = plan_ticket; pa.err = err;
    const int plan_grid = 1 + (B + kPlanThreads / 32 - 1) / (kPlanThreads / 32);
    if (eti_launch_pdl(decode_plan_kernel, dim3(plan_grid), dim3(kPlanThreads), 0, stream, pa) != cudaSuccess)
        return ETI_ERR_CUDA;

    DecArgs da;
    da.v_cache = v_cache; da.block_table = block_table; da.ctx_lens = ctx_lens;
    da.kept_idx = kept_idx; da.token_scores = token_scores; da.kept_norm = kept_norm;
    da.cum = plan_cum; da.info = plan_info; da.warp_seg = plan_warp_seg;
    da.B = B; da.Hq = Hq; da.Hkv = Hkv; da.g = Hq / Hkv; da.max_blocks = max_blocks;
    da.num_pages = num_pages; da.out = out; da.partial = partial;
    da.ticket = plan_ticket; da.err = err;
    da.wait_iters = eti_wait_limit();
    const int grid = nwarps / kDecWarps;
    if (num_pages <= 0 || num_pages * Hkv * P >= (1LL << 31)) {
        if (num_pages > 0) return ETI_ERR_UNSUPPORTED;   // tile rows are int32 on the device
    }
    CUtensorMap vmap;
    if (num_pages > 0) {
        const int st = eti_make_kv_tensor_map(&vmap, v_cache, num_pages * Hkv * P, D);
        if (st != ETI_OK) return st;
    } else {
        memset(&vmap, 0, sizeof(vmap));   // no page is valid: the kernel issues no copy
    }
    bool launched = false;
#define ETI_DEC_CASE(DD, PP)                                                              \
    if (!launched && D == DD && P == PP) {                                                \
        auto k = paged_decode_kernel<DD, PP>;                                             \
        const size_t sm = dec_smem_bytes<DD>(Hq / Hkv);                                   \
        cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);    \
        if (eti_launch_pdl(k, dim3(grid), dim3(kDecThreads), sm, stream, vmap, da) != cudaSuccess) \
            return ETI_ERR_CUDA;                                                          \
        launched = true;                                                                  \
    }
    ETI_DEC_CASE(128, 16)
    ETI_DEC_CASE(128, 32)
    ETI_DEC_CASE(64, 16)
    ETI_DEC_CASE(64, 32)
#undef ETI_DEC_CASE
    if (!launched) return ETI_ERR_UNSUPPORTED;
    return cudaGetLastError() == cudaSuccess ? ETI_OK : ETI_ERR_CUDA;
}
