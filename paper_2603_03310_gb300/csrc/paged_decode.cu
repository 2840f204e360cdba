// paged_decode.cu -- GQA paged decode attention restricted to the kept blocks
// (Section 3.2: attention is computed over B_t only, renormalised over the
// kept tokens).
//
// The scorer already produced x_i = scale q_h . k_i for every token and the
// finalizer the kept-token softmax normaliser (M_h, l_h) of every query head,
// so this pass reads only the kept V pages and their scores:
//   out_h = (1 / l_h) sum_{i kept} e^{x_i - M_h} v_i .
// Because the weights are already normalised against a fixed M_h, partial
// sums over different block ranges simply add (no rescaling).
//
// Work split (stream-K over kept blocks): the kept blocks of all (sequence,
// kv head) segments form one list; CTA c takes the contiguous range
// [c*share, (c+1)*share).  Inside a CTA the 8 warps take the blocks of a
// segment round-robin, each accumulating p.V with bf16 m16n8k16 tensor-core
// tiles (head_dim = M, query heads = N, tokens = K): a thread's 128-bit loads
// of V rows are transposed into A fragments with byte permutes, the
// probabilities form the B fragment.  Warps are reduced through shared
// memory at the end of each segment piece; a segment that one CTA covers is
// written straight to `out`, otherwise the piece goes to partial slot
// (c + segment) and the combine kernel adds the slots in CTA order.
#include "common.cuh"

namespace eti {

constexpr int kDecThreads = 256;
constexpr int kDecWarps = kDecThreads / 32;
constexpr int kPlanThreads = 1024;

// --------------------------------------------------------------------------
// plan: prefix of kept counts, the per-CTA share and each CTA's first segment
struct PlanArgs {
    const int32_t* kept_cnt;
    int nseg, ncta, max_blocks;
    int* cum;       // [nseg + 1]
    int* info;      // [0] = total kept blocks, [1] = share
    int* cta_seg;   // [ncta]
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
    const int share = max(1, (total + a.ncta - 1) / a.ncta);
    if (tid == 0) {
        a.cum[a.nseg] = total;
        a.info[0] = total;
        a.info[1] = share;
    }
    for (int c = tid; c < a.ncta; c += kPlanThreads) a.cta_seg[c] = a.nseg;
    __syncthreads();
    for (int s = tid; s < a.nseg; s += kPlanThreads) {
        const int lo = a.cum[s], hi = a.cum[s + 1];
        if (hi <= lo) continue;
        const int c0 = (lo + share - 1) / share, c1 = min((hi + share - 1) / share, a.ncta);
        for (int c = c0; c < c1; ++c) a.cta_seg[c] = s;
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
    const int* cta_seg;
    int B, Hq, Hkv, g, max_blocks;
    long long num_pages;
    uint16_t* out;                 // bf16 [B][Hq][D]
    float* partial;                // [(ncta + nseg)][g][D]
};

template <int D>
struct VTile {
    static constexpr int kElems = D / 16;              // elements per row half per thread
    using Vec = typename std::conditional<kElems == 8, uint4, uint2>::type;
    Vec r[4][2];                                       // rows 2t, 2t+1, 2t+8, 2t+9; halves
    float x[4];                                        // scores of those rows, head grp
};

template <int D>
__device__ __forceinline__ uint32_t vreg(const typename VTile<D>::Vec& v, int i) {
    if constexpr (VTile<D>::kElems == 8) {
        return i == 0 ? v.x : i == 1 ? v.y : i == 2 ? v.z : v.w;
    } else {
        return i == 0 ? v.x : v.y;
    }
}

// bf16 element j of rows (ra, rb) packed as (ra.j, rb.j)
template <int D>
__device__ __forceinline__ uint32_t pair_elem(const typename VTile<D>::Vec& ra,
                                              const typename VTile<D>::Vec& rb, int j) {
    const uint32_t a = vreg<D>(ra, j >> 1), b = vreg<D>(rb, j >> 1);
    return (j & 1) ? hi_halves(a, b) : lo_halves(a, b);
}

template <int D>
__device__ __forceinline__ typename VTile<D>::Vec ld_vec(const uint16_t* p) {
    if constexpr (VTile<D>::kElems == 8) return ldg_stream_u4(p);
    else return ldg_stream_u2(p);
}

template <int D>
__device__ __forceinline__ typename VTile<D>::Vec zero_vec() {
    typename VTile<D>::Vec z;
    if constexpr (VTile<D>::kElems == 8) z = make_uint4(0, 0, 0, 0);
    else z = make_uint2(0, 0);
    return z;
}

// rows of the A fragment owned by a thread (tq = lane & 3)
__device__ __forceinline__ int frag_row(int tq, int k) { return 2 * tq + (k & 1) + (k >> 1) * 8; }

template <int D, int P>
__device__ __forceinline__ void load_v_tile(VTile<D>& t, const DecArgs& a, long long unit,
                                            const uint16_t* vtile, int tile, int valid_tok,
                                            bool valid, int grp, int tq) {
    constexpr int E = VTile<D>::kElems;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const int row = frag_row(tq, k);
        const bool ok = valid && (tile * 16 + row) < valid_tok;
        if (ok) {
            t.r[k][0] = ld_vec<D>(vtile + row * D + E * grp);
            t.r[k][1] = ld_vec<D>(vtile + row * D + D / 2 + E * grp);
            t.x[k] = grp < a.g ? __ldg(a.token_scores + (unit * P + tile * 16 + row) * a.g + grp) : -kInf;
        } else {
            t.r[k][0] = zero_vec<D>();
            t.r[k][1] = zero_vec<D>();
            t.x[k] = -kInf;
        }
    }
}

template <int D, int P>
__global__ void __launch_bounds__(kDecThreads, 2)
paged_decode_kernel(const DecArgs a) {
    constexpr int kTiles = P / 16;
    constexpr int J = D / 16;                      // MMAs per 16-token tile
    __shared__ float red[kDecWarps][8][D];
    const int total = a.info[0], share = a.info[1];
    const int c = blockIdx.x;
    int u0 = c * share;
    const int u1 = min(u0 + share, total);
    if (u0 >= u1) return;
    int s = a.cta_seg[c];
    const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5, grp = lane >> 2, tq = lane & 3;

    while (u0 < u1 && s < a.Hkv * a.B) {
        const int seg_lo = a.cum[s], seg_hi = a.cum[s + 1];
        if (seg_hi <= u0) { ++s; continue; }
        const int p1 = min(u1, seg_hi);
        const int i0 = u0 - seg_lo, i1 = p1 - seg_lo;
        const bool whole = (u0 == seg_lo) && (p1 == seg_hi);
        const int b = s / a.Hkv, kvh = s - b * a.Hkv;
        const int L = a.ctx_lens[b];
        const int nb = seq_blocks(L, P, a.max_blocks);
        const float Mh = grp < a.g ? a.kept_norm[((long long)b * a.Hq + kvh * a.g + grp) * 2] : 0.f;

        float acc[J][4];
#pragma unroll
        for (int j = 0; j < J; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;

        // this warp's tiles: items i0 + w + 8 k, tiles 0..kTiles-1 each
        const int nitems = i1 - i0 > w ? (i1 - i0 - w + kDecWarps - 1) / kDecWarps : 0;
        const int ntiles = nitems * kTiles;
        auto tile_src = [&](int step, long long& unit, const uint16_t*& vt, int& tile, int& vtok,
                            bool& valid) {
            const int item = i0 + w + (step / kTiles) * kDecWarps;
            tile = step - (step / kTiles) * kTiles;
            const int blk = a.kept_idx[(long long)s * a.max_blocks + item];
            valid = blk >= 0 && blk < nb;
            const int page = valid ? a.block_table[(long long)b * a.max_blocks + blk] : 0;
            valid = valid && page >= 0 && (long long)page < a.num_pages;
            unit = (long long)s * a.max_blocks + (valid ? blk : 0);
            vtok = valid ? min(P, L - blk * P) : 0;
            vt = a.v_cache + ((long long)(valid ? page : 0) * a.Hkv + kvh) * P * D + tile * 16 * D;
        };
        auto consume = [&](const VTile<D>& t) {
            float p[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) p[k] = fast_ex2((t.x[k] - Mh) * kLog2e);
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
        if (ntiles > 0) {
            VTile<D> t0, t1;
            {
                long long unit; const uint16_t* vt; int tile, vtok; bool valid;
                tile_src(0, unit, vt, tile, vtok, valid);
                load_v_tile<D, P>(t0, a, unit, vt, tile, vtok, valid, grp, tq);
            }
            for (int st = 0; st < ntiles; st += 2) {
                if (st + 1 < ntiles) {
                    long long unit; const uint16_t* vt; int tile, vtok; bool valid;
                    tile_src(st + 1, unit, vt, tile, vtok, valid);
                    load_v_tile<D, P>(t1, a, unit, vt, tile, vtok, valid, grp, tq);
                }
                consume(t0);
                if (st + 1 < ntiles) {
                    if (st + 2 < ntiles) {
                        long long unit; const uint16_t* vt; int tile, vtok; bool valid;
                        tile_src(st + 2, unit, vt, tile, vtok, valid);
                        load_v_tile<D, P>(t0, a, unit, vt, tile, vtok, valid, grp, tq);
                    }
                    consume(t1);
                }
            }
        }
        // reduce the 8 warps: head n = 2tq + (e & 1); d from the fragment row
#pragma unroll
        for (int j = 0; j < J; ++j) {
            const int d_lo = J * grp + j, d_hi = D / 2 + J * grp + j;
            red[w][2 * tq][d_lo] = acc[j][0];
            red[w][2 * tq + 1][d_lo] = acc[j][1];
            red[w][2 * tq][d_hi] = acc[j][2];
            red[w][2 * tq + 1][d_hi] = acc[j][3];
        }
        __syncthreads();
        for (int e = tid; e < a.g * D; e += kDecThreads) {
            const int h = e / D, d = e - h * D;
            float v = 0.f;
#pragma unroll
            for (int ww = 0; ww < kDecWarps; ++ww) v += red[ww][h][d];
            if (whole) {
                const float l = a.kept_norm[((long long)b * a.Hq + kvh * a.g + h) * 2 + 1];
                const float o = l > 0.f ? v / l : 0.f;
                a.out[((long long)b * a.Hq + kvh * a.g + h) * D + d] = __bfloat16_as_ushort(__float2bfloat16_rn(o));
            } else {
                a.partial[((long long)(c + s) * a.g + h) * D + d] = v;
            }
        }
        __syncthreads();
        u0 = p1;
        if (p1 == seg_hi) ++s;
    }
}

// --------------------------------------------------------------------------
// combine: add the partial slots of segments split across CTAs; zero the
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
    const int c0 = lo / share, c1 = (hi - 1) / share;
    if (c0 == c1) return;   // one CTA covered the segment and wrote it
    for (int e = tid; e < a.g * a.D; e += blockDim.x) {
        const int h = e / a.D, d = e - h * a.D;
        float v = 0.f;
        for (int c = c0; c <= c1; ++c) v += a.partial[((long long)(c + s) * a.g + h) * a.D + d];
        const float l = a.kept_norm[((long long)b * a.Hq + kvh * a.g + h) * 2 + 1];
        o[e] = __bfloat16_as_ushort(__float2bfloat16_rn(l > 0.f ? v / l : 0.f));
    }
}

}  // namespace eti

using namespace eti;

int eti_decode_ncta() {
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    return 2 * sms;
}

int eti_launch_decode(const uint16_t* v_cache, const int32_t* block_table, const int32_t* ctx_lens,
                      const int32_t* kept_idx, const int32_t* kept_cnt, const float* token_scores,
                      const float* kept_norm, int B, int Hq, int Hkv, int D, int P, int max_blocks,
                      long long num_pages, uint16_t* out, uint32_t* err, int* plan_cum,
                      int* plan_info, int* plan_cta_seg, float* partial, int ncta,
                      cudaStream_t stream) {
    if (B == 0) return ETI_OK;
    const int nseg = B * Hkv;
    PlanArgs pa;
    pa.kept_cnt = kept_cnt; pa.nseg = nseg; pa.ncta = ncta; pa.max_blocks = max_blocks;
    pa.cum = plan_cum; pa.info = plan_info; pa.cta_seg = plan_cta_seg;
    decode_plan_kernel<<<1, kPlanThreads, 0, stream>>>(pa);
    if (cudaGetLastError() != cudaSuccess) return ETI_ERR_CUDA;

    DecArgs da;
    da.v_cache = v_cache; da.block_table = block_table; da.ctx_lens = ctx_lens;
    da.kept_idx = kept_idx; da.token_scores = token_scores; da.kept_norm = kept_norm;
    da.cum = plan_cum; da.info = plan_info; da.cta_seg = plan_cta_seg;
    da.B = B; da.Hq = Hq; da.Hkv = Hkv; da.g = Hq / Hkv; da.max_blocks = max_blocks;
    da.num_pages = num_pages; da.out = out; da.partial = partial;
    bool launched = false;
#define ETI_DEC_CASE(DD, PP)                                                        \
    if (!launched && D == DD && P == PP) {                                          \
        paged_decode_kernel<DD, PP><<<ncta, kDecThreads, 0, stream>>>(da);          \
        launched = true;                                                            \
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
