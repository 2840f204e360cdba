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
// [w*share, (w+1)*share).  Each warp loads its 16-token tiles straight into
// registers with 128-bit loads, one tile ahead of use, and keeps a deeper
// stream in flight with bulk L2 prefetches (one instruction per kept V chunk)
// a few blocks further ahead.  Page ids are resolved 32 blocks at a time, one
// lane per block, a batch ahead of use.  p.V runs on bf16 m16n8k16 tensor-core tiles
// (head_dim = M, query heads = N, tokens = K): V rows are transposed into A
// fragments with byte permutes, the probabilities form the B fragment.
// A segment that lies inside one warp's range is written straight to `out`;
// otherwise the warp's part goes to partial slot (warp + segment) and the
// combine kernel adds the slots in warp order (deterministic).
#include "common.cuh"

namespace eti {

constexpr int kDecWarps = 8;
constexpr int kDecThreads = kDecWarps * 32;
constexpr int kPlanThreads = 1024;

// --------------------------------------------------------------------------
// plan: prefix of kept counts, the per-warp share and each warp's first segment
struct PlanArgs {
    const int32_t* kept_cnt;
    int nseg, nwarps, max_blocks;
    int* cum;       // [nseg + 1]
    int* info;      // [0] = total kept blocks, [1] = share per warp
    int* warp_seg;  // [nwarps]
};

__global__ void __launch_bounds__(kPlanThreads) decode_plan_kernel(const PlanArgs a) {
    __shared__ int wsum[kPlanThreads / 32];
    const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
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
        if (s < a.nseg) a.cum[s] = carry + ofs + x - v;
        carry += tot;
        __syncthreads();
    }
    const int total = carry;
    const int share = max(1, (total + a.nwarps - 1) / a.nwarps);
    if (tid == 0) {
        a.cum[a.nseg] = total;
        a.info[0] = total;
        a.info[1] = share;
    }
    for (int c = tid; c < a.nwarps; c += kPlanThreads) a.warp_seg[c] = a.nseg;
    __syncthreads();
    for (int s = tid; s < a.nseg; s += kPlanThreads) {
        const int lo = a.cum[s], hi = a.cum[s + 1];
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
};

constexpr int kDecPrefetch = 6;    // kept blocks prefetched into L2 ahead of the loads

template <int D>
struct DecLayout {
    static constexpr int E = D / 16;              // bf16 per row half per thread
    using Vec = typename std::conditional<E == 8, uint4, uint2>::type;
};

template <int D>
__device__ __forceinline__ uint32_t vreg(const typename DecLayout<D>::Vec& v, int i) {
    if constexpr (DecLayout<D>::E == 8) {
        return i == 0 ? v.x : i == 1 ? v.y : i == 2 ? v.z : v.w;
    } else {
        return i == 0 ? v.x : v.y;
    }
}

// bf16 element j of rows (ra, rb) packed as (ra.j, rb.j)
template <int D>
__device__ __forceinline__ uint32_t pair_elem(const typename DecLayout<D>::Vec& ra,
                                              const typename DecLayout<D>::Vec& rb, int j) {
    const uint32_t x = vreg<D>(ra, j >> 1), y = vreg<D>(rb, j >> 1);
    return (j & 1) ? hi_halves(x, y) : lo_halves(x, y);
}

template <int D>
__device__ __forceinline__ typename DecLayout<D>::Vec ld_vec(const uint16_t* p) {
    if constexpr (DecLayout<D>::E == 8) return ldg_stream_u4(p);
    else return ldg_stream_u2(p);
}

template <int D>
__device__ __forceinline__ typename DecLayout<D>::Vec zero_vec() {
    typename DecLayout<D>::Vec z;
    if constexpr (DecLayout<D>::E == 8) z = make_uint4(0, 0, 0, 0);
    else z = make_uint2(0, 0);
    return z;
}

// A-fragment rows owned by a thread (tq = lane & 3): 2tq, 2tq+1, 2tq+8, 2tq+9
__device__ __forceinline__ int frag_row(int tq, int k) { return 2 * tq + (k & 1) + (k >> 1) * 8; }

// one block of the warp's range, resolved by one lane
struct ItemInfo {
    int seg, blk, page, vtok;
};

template <int D>
struct VTile {
    typename DecLayout<D>::Vec r[4][2];   // rows 2t, 2t+1, 2t+8, 2t+9; halves
    float x[4];                           // their scores for head grp
    int seg;
};

template <int D, int P>
__global__ void __launch_bounds__(kDecThreads, 1)
paged_decode_kernel(const DecArgs a) {
    using LY = DecLayout<D>;
    constexpr int kTiles = P / 16;
    constexpr int J = D / 16;                    // MMAs per 16-token tile
    const int lane = threadIdx.x & 31, wl = threadIdx.x >> 5, grp = lane >> 2, tq = lane & 3;
    const int warp = blockIdx.x * kDecWarps + wl;
    const int total = a.info[0], share = a.info[1];
    const int u0 = warp * share;
    const int u1 = min(u0 + share, total);
    if (u0 >= u1) return;
    const int nseg = a.B * a.Hkv;
    const int ntiles = (u1 - u0) * kTiles;

    auto resolve = [&](int base, int seg_hint) -> ItemInfo {
        ItemInfo it{seg_hint, 0, -1, 0};
        const int u = base + lane;
        if (u < u1) {
            int s = seg_hint;
            while (s < nseg - 1 && __ldg(a.cum + s + 1) <= u) ++s;
            it.seg = s;
            const int b = s / a.Hkv;
            const int L = __ldg(a.ctx_lens + b);
            const int nb = seq_blocks(L, P, a.max_blocks);
            const int blk = __ldg(a.kept_idx + (long long)s * a.max_blocks + (u - __ldg(a.cum + s)));
            if (blk >= 0 && blk < nb) {
                const int pg = __ldg(a.block_table + (long long)b * a.max_blocks + blk);
                if (pg >= 0 && (long long)pg < a.num_pages) {
                    it.blk = blk;
                    it.page = pg;
                    it.vtok = min(P, L - blk * P);
                }
            }
        }
        return it;
    };

    ItemInfo cur = resolve(u0, a.warp_seg[warp]);
    int cbase = u0;
    ItemInfo nxt = resolve(u0 + 32, __shfl_sync(0xffffffffu, cur.seg, 31));
    auto item_at = [&](int off) -> ItemInfo {
        const int l = off & 31;
        ItemInfo a0, a1;
        a0.seg = __shfl_sync(0xffffffffu, cur.seg, l);   a1.seg = __shfl_sync(0xffffffffu, nxt.seg, l);
        a0.blk = __shfl_sync(0xffffffffu, cur.blk, l);   a1.blk = __shfl_sync(0xffffffffu, nxt.blk, l);
        a0.page = __shfl_sync(0xffffffffu, cur.page, l); a1.page = __shfl_sync(0xffffffffu, nxt.page, l);
        a0.vtok = __shfl_sync(0xffffffffu, cur.vtok, l); a1.vtok = __shfl_sync(0xffffffffu, nxt.vtok, l);
        return off < 32 ? a0 : a1;
    };
    auto v_chunk = [&](const ItemInfo& it) {
        const int kvh = it.seg - (it.seg / a.Hkv) * a.Hkv;
        return a.v_cache + ((long long)(it.page >= 0 ? it.page : 0) * a.Hkv + kvh) * P * D;
    };
    auto s_chunk = [&](const ItemInfo& it) {
        return a.token_scores + ((long long)it.seg * a.max_blocks + it.blk) * P * a.g;
    };
    auto prefetch = [&](const ItemInfo& it) {
        if (lane == 0 && it.page >= 0) {
            prefetch_l2_bulk(v_chunk(it), P * D * 2);
            if (((P * a.g * 4) & 15) == 0) prefetch_l2_bulk(s_chunk(it), P * a.g * 4);
        }
    };
    auto load_tile = [&](VTile<D>& t, const ItemInfo& it, int tile) {
        const uint16_t* vt = v_chunk(it) + tile * 16 * D;
        const float* sc = s_chunk(it) + tile * 16 * a.g;
        const bool ok = it.page >= 0;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int row = frag_row(tq, k);
            if (ok && tile * 16 + row < it.vtok) {
                t.r[k][0] = ld_vec<D>(vt + row * D + LY::E * grp);
                t.r[k][1] = ld_vec<D>(vt + row * D + D / 2 + LY::E * grp);
                t.x[k] = grp < a.g ? __ldg(sc + row * a.g + grp) : 0.f;
            } else {
                t.r[k][0] = zero_vec<D>();
                t.r[k][1] = zero_vec<D>();
                t.x[k] = 0.f;
            }
        }
        t.seg = it.seg;
    };

    for (int k = 0; k < kDecPrefetch && u0 + k < u1; ++k) prefetch(item_at(k));

    float acc[J][4];
#pragma unroll
    for (int j = 0; j < J; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;

    // write the accumulated segment: straight to `out` when the whole segment
    // is in this warp's range, else into partial slot (warp + seg)
    auto flush = [&](int seg) {
        const int b = seg / a.Hkv, kvh = seg - b * a.Hkv;
        const int lo = __ldg(a.cum + seg), hi = __ldg(a.cum + seg + 1);
        const bool whole = lo >= u0 && hi <= u1;
#pragma unroll
        for (int e = 0; e < 2; ++e) {
            const int h = 2 * tq + e;
            if (h < a.g) {
#pragma unroll
                for (int half = 0; half < 2; ++half) {
                    const int d0 = half * (D / 2) + J * grp;
                    float v[J];
#pragma unroll
                    for (int j = 0; j < J; ++j) v[j] = acc[j][2 * half + e];
                    if (whole) {
                        const float l = __ldg(a.kept_norm + ((long long)b * a.Hq + kvh * a.g + h) * 2 + 1);
                        const float inv = l > 0.f ? 1.f / l : 0.f;
                        uint32_t pk[J / 2];
#pragma unroll
                        for (int j = 0; j < J / 2; ++j) pk[j] = pack_bf16x2(v[2 * j] * inv, v[2 * j + 1] * inv);
                        uint16_t* o = a.out + ((long long)b * a.Hq + kvh * a.g + h) * D + d0;
                        if constexpr (J == 8) *reinterpret_cast<uint4*>(o) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
                        else *reinterpret_cast<uint2*>(o) = make_uint2(pk[0], pk[1]);
                    } else {
                        float* o = a.partial + ((long long)(warp + seg) * a.g + h) * D + d0;
#pragma unroll
                        for (int j = 0; j < J; j += 4)
                            *reinterpret_cast<float4*>(o + j) = make_float4(v[j], v[j + 1], v[j + 2], v[j + 3]);
                    }
                }
            }
        }
#pragma unroll
        for (int j = 0; j < J; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;
    };

    int cur_seg = -1;
    float Mh = 0.f;
    // consume one tile: probabilities (B fragment) and p.V on the tensor cores
    auto consume = [&](const VTile<D>& t) {
        if (t.seg != cur_seg) {
            if (cur_seg >= 0) flush(cur_seg);
            cur_seg = t.seg;
            const int b = cur_seg / a.Hkv, kvh = cur_seg - b * a.Hkv;
            Mh = grp < a.g ? __ldg(a.kept_norm + ((long long)b * a.Hq + kvh * a.g + grp) * 2) : 0.f;
        }
        float p[4];
#pragma unroll
        for (int k = 0; k < 4; ++k)
            // kept tokens have x <= M_h; zeroed rows (past the end, or a padded
            // head) get weight 1 against a zero V row
            p[k] = fast_ex2(fminf((t.x[k] - Mh) * kLog2e, 0.f));
        const uint32_t b0 = pack_bf16x2(p[0], p[1]);
        const uint32_t b1 = pack_bf16x2(p[2], p[3]);
#pragma unroll
        for (int j = 0; j < J; ++j) {
            const uint32_t a0 = pair_elem<D>(t.r[0][0], t.r[1][0], j);
            const uint32_t a1 = pair_elem<D>(t.r[0][1], t.r[1][1], j);
            const uint32_t a2 = pair_elem<D>(t.r[2][0], t.r[3][0], j);
            const uint32_t a3 = pair_elem<D>(t.r[2][1], t.r[3][1], j);
            mma_bf16_16x8x16(acc[j], a0, a1, a2, a3, b0, b1);
        }
    };

    // next tile i + 1: load it (and prefetch further ahead into L2)
    auto advance = [&](VTile<D>& t, int i) {
        const int item = u0 + i / kTiles;
        const int tile = i - (i / kTiles) * kTiles;
        if (item >= cbase + 32) {
            cur = nxt;
            cbase += 32;
            nxt = resolve(cbase + 32, __shfl_sync(0xffffffffu, cur.seg, 31));
        }
        load_tile(t, item_at(item - cbase), tile);
        if (tile == 0 && item + kDecPrefetch < u1) prefetch(item_at(item + kDecPrefetch - cbase));
    };

    VTile<D> t0, t1;
    load_tile(t0, item_at(0), 0);
    for (int i = 0; i < ntiles; i += 2) {
        if (i + 1 < ntiles) advance(t1, i + 1);
        consume(t0);
        if (i + 1 < ntiles) {
            if (i + 2 < ntiles) advance(t0, i + 2);
            consume(t1);
        }
    }
    if (cur_seg >= 0) flush(cur_seg);
}

// --------------------------------------------------------------------------
// combine: add the partial slots of segments split across warps; zero the
// output of segments with nothing kept or of invalid sequences.
struct CombArgs {
    const int* cum;
    const int* info;
    const float* partial;
    const float* kept_norm;
    const int32_t* ctx_lens;
    const int32_t* block_table;
    long long num_pages;
    int B, Hq, Hkv, g, D, P, max_blocks;
    uint16_t* out;
    uint32_t* err;
};

__global__ void __launch_bounds__(128) decode_combine_kernel(const CombArgs a) {
    const int s = blockIdx.x;
    const int b = s / a.Hkv, kvh = s - b * a.Hkv;
    const int tid = threadIdx.x;
    const int L = a.ctx_lens[b];
    const bool bad_ctx = L < 0 || L > a.max_blocks * a.P;
    const int nb = bad_ctx ? 0 : (L + a.P - 1) / a.P;
    int bad = 0;
    for (int j = tid; j < nb; j += blockDim.x) {
        const int pg = a.block_table[(long long)b * a.max_blocks + j];
        bad |= (pg < 0 || (long long)pg >= a.num_pages);
    }
    const bool bad_page = __syncthreads_or(bad) != 0;
    if (a.err && kvh == 0 && tid == 0)
        a.err[b] = bad_ctx ? ETI_ERRF_BAD_CTX : (bad_page ? ETI_ERRF_BAD_PAGE : 0u);
    const int lo = a.cum[s], hi = a.cum[s + 1];
    const int share = a.info[1];
    uint16_t* o = a.out + ((long long)b * a.Hq + kvh * a.g) * a.D;
    if (bad_ctx || bad_page || hi <= lo) {
        for (int e = tid; e < a.g * a.D; e += blockDim.x) o[e] = 0;
        return;
    }
    const int w0 = lo / share, w1 = (hi - 1) / share;
    if (w0 == w1) return;   // one warp covered the segment and wrote it
    for (int e = tid; e < a.g * a.D; e += blockDim.x) {
        const int h = e / a.D, d = e - h * a.D;
        float v = 0.f;
        for (int w = w0; w <= w1; ++w) v += a.partial[((long long)(w + s) * a.g + h) * a.D + d];
        const float l = a.kept_norm[((long long)b * a.Hq + kvh * a.g + h) * 2 + 1];
        o[e] = __bfloat16_as_ushort(__float2bfloat16_rn(l > 0.f ? v / l : 0.f));
    }
}

}  // namespace eti

using namespace eti;

// warps of the persistent decode grid on the current device
int eti_decode_nwarps() {
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    return sms * kDecWarps;
}

int eti_launch_decode(const uint16_t* v_cache, const int32_t* block_table, const int32_t* ctx_lens,
                      const int32_t* kept_idx, const int32_t* kept_cnt, const float* token_scores,
                      const float* kept_norm, int B, int Hq, int Hkv, int D, int P, int max_blocks,
                      long long num_pages, uint16_t* out, uint32_t* err, int* plan_cum,
                      int* plan_info, int* plan_warp_seg, float* partial, int nwarps,
                      cudaStream_t stream) {
    if (B == 0) return ETI_OK;
    const int nseg = B * Hkv;
    PlanArgs pa;
    pa.kept_cnt = kept_cnt; pa.nseg = nseg; pa.nwarps = nwarps; pa.max_blocks = max_blocks;
    pa.cum = plan_cum; pa.info = plan_info; pa.warp_seg = plan_warp_seg;
    decode_plan_kernel<<<1, kPlanThreads, 0, stream>>>(pa);
    if (cudaGetLastError() != cudaSuccess) return ETI_ERR_CUDA;

    DecArgs da;
    da.v_cache = v_cache; da.block_table = block_table; da.ctx_lens = ctx_lens;
    da.kept_idx = kept_idx; da.token_scores = token_scores; da.kept_norm = kept_norm;
    da.cum = plan_cum; da.info = plan_info; da.warp_seg = plan_warp_seg;
    da.B = B; da.Hq = Hq; da.Hkv = Hkv; da.g = Hq / Hkv; da.max_blocks = max_blocks;
    da.num_pages = num_pages; da.out = out; da.partial = partial;
    const int grid = nwarps / kDecWarps;
    bool launched = false;
#define ETI_DEC_CASE(DD, PP)                                                              \
    if (!launched && D == DD && P == PP) {                                                \
        paged_decode_kernel<DD, PP><<<grid, kDecThreads, 0, stream>>>(da);                \
        launched = true;                                                                  \
    }
    ETI_DEC_CASE(128, 16)
    ETI_DEC_CASE(128, 32)
    ETI_DEC_CASE(64, 16)
    ETI_DEC_CASE(64, 32)
#undef ETI_DEC_CASE
    if (!launched) return ETI_ERR_UNSUPPORTED;
    if (cudaGetLastError() != cudaSuccess) return ETI_ERR_CUDA;

    CombArgs ca;
    ca.cum = plan_cum; ca.info = plan_info; ca.partial = partial; ca.kept_norm = kept_norm;
    ca.ctx_lens = ctx_lens; ca.block_table = block_table; ca.num_pages = num_pages;
    ca.B = B; ca.Hq = Hq; ca.Hkv = Hkv; ca.g = Hq / Hkv; ca.D = D; ca.P = P;
    ca.max_blocks = max_blocks; ca.out = out; ca.err = err;
    decode_combine_kernel<<<nseg, 128, 0, stream>>>(ca);
    return cudaGetLastError() == cudaSuccess ? ETI_OK : ETI_ERR_CUDA;
}
