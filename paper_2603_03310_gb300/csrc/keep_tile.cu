// keep_tile.cu -- the keep set of segments of up to kTileItems block-heads
// (Section 3.2: the block entropy terms I_b, the block scores, the threshold
// / budget rule, compaction, the softmax normaliser over the kept tokens),
// one CTA of NW warps per (sequence, kv head) segment.
//
// Warp w owns a contiguous range of the segment's blocks: it stages their
// block stats (g float4 a block) in shared memory with cp.async and takes, in
// rounds, query head h = l % GP of the blocks l / GP + r (32 / GP) of its
// range (lane l, GP the power of two >= g).  Per-head sums are shuffle
// butterflies over the lanes of equal head, then NW partials in shared
// memory; the kept blocks are ranked by ballots in ascending block order
// within a warp and by the warps' counts across them.  The work follows the
// segment's length (not max_blocks) and three CTA barriers separate the
// passes over the staged stats:
//   A  the head's max M = max_b m_b (and the timeout marks of the scorer);
//   B  c_b = e^{m_b - M}, z_b = c_b (1 + l1_b); the sums Z - 1, A = sum z_b
//      (M - m_b) and U = sum c_b u_b give H = log Z + (A - U) / Z, the sum of
//      the block terms; (z_b, c_b u_b) replace (l1_b, u_b) in shared memory;
//   C  I_b = [z_b (log Z + M - m_b) - c_b u_b] / Z, the group score (the
//      largest n_b I_b / H over the heads of the block), the threshold's
//      kept count and the argmax block of each warp;
//   D  keep decisions and compaction (the B_min > 1 budget: a radix select
//      of the kb-th score key by warp 0, which then ranks every block);
//   E  (M_k, L_k) of each head over the kept blocks: the z_b sums against M,
//      taken again against M_k from the stats when the block holding a
//      head's largest logit was left out.
#include "keep_set.cuh"

namespace eti {

constexpr int kTileItems = 8192;        // largest max_blocks * g the kernel stages

// shared memory of a CTA: the radix histogram, the stats, the block scores,
// the keep flags
inline size_t tile_smem(int max_blocks, int g) {
    return (1024 + (size_t)max_blocks * g * 16 + (size_t)max_blocks * 5 + 15) / 16 * 16;
}

template <int G, int NW>
__global__ void __launch_bounds__(NW * 32) prune_finalize_tile_kernel(const FinArgs a) {
    constexpr int GP = FlatGP<G>::v;
    constexpr int BR = 32 / GP;                  // blocks of a round
    constexpr int NT = NW * 32;
    constexpr unsigned kAll = 0xffffffffu;
    pdl_trigger();
    pdl_wait();
    extern __shared__ __align__(16) unsigned char tile_smem_raw[];
    int* hist = reinterpret_cast<int*>(tile_smem_raw);
    float4* sm = reinterpret_cast<float4*>(tile_smem_raw + 1024);
    float* sc = reinterpret_cast<float*>(tile_smem_raw + 1024 + (size_t)a.max_blocks * G * 16);
    uint8_t* kf = reinterpret_cast<uint8_t*>(sc + a.max_blocks);
    __shared__ float red_m[NW][GP];
    __shared__ float4 red_s[NW][GP];
    __shared__ unsigned red_f[NW];
    __shared__ float arg_v[NW];
    __shared__ int arg_j[NW], cnt[NW];
    __shared__ float kn_m[NW][GP], kn_l[NW][GP];
    __shared__ int sel[2];
    const int b = blockIdx.x, kvh = blockIdx.y;  // grid (B, Hkv)
    const int seg = b * a.Hkv + kvh;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int h = lane & (GP - 1), jr = lane / GP;
    const bool hv = h < G;
    const int L = a.ctx_lens[b];
    const float th = a.theta[b];
    const bool bad_ctx = L < 0 || L > a.max_blocks * a.P;
    const int nb = bad_ctx ? 0 : (L + a.P - 1) / a.P;
    const long long segbase = (long long)seg * a.max_blocks;
    const float4* st = a.stats + segbase * G;
    // warp w owns blocks [j0, j1): contiguous ranges in block order, whole rounds
    const int q = ((nb + NW - 1) / NW + BR - 1) / BR * BR;
    const int j0 = min(nb, wid * q), j1 = min(nb, j0 + q);

    // stage the warp's stats; check its page ids meanwhile
    const uint32_t sbase = smem_u32(sm);
    for (int i = j0 * G + lane; i < j1 * G; i += 32) cp_async_16(sbase + i * 16, st + i, true);
    cp_async_commit();
    const bool bad = any_bad_page(a.block_table + (long long)b * a.max_blocks, j0 + lane, 32, j1, a.num_pages);
    cp_async_wait<0>();
    __syncwarp();

    // A: the head's max; a NaN max marks a block the scoring pass gave up on
    // (l - 1 = +inf: and the drain of its copies gave up too)
    float M = -kInf;
    bool stale = false, drain = false;
    for (int j = j0 + jr; j < j1; j += BR)
        if (hv) {
            const float4 s = sm[j * G + h];
            M = fmaxf(M, s.x);
            stale |= s.x != s.x;
            drain |= s.x != s.x && s.y == kInf;
        }
#pragma unroll
    for (int o = GP; o < 32; o <<= 1) M = fmaxf(M, __shfl_xor_sync(kAll, M, o));
    const unsigned fl = __reduce_or_sync(kAll, (bad ? 1u : 0u) | (stale ? 2u : 0u) | (drain ? 4u : 0u));
    if (lane < GP) red_m[wid][lane] = M;
    if (lane == 0) red_f[wid] = fl;
    __syncthreads();
    unsigned flags = 0;
#pragma unroll
    for (int u = 0; u < NW; ++u) { flags |= red_f[u]; M = fmaxf(M, red_m[u][h]); }
    const bool bad_page = (flags & 1u) != 0;
    const bool timed_out = (flags & 2u) && !bad_page;
    if (a.err && tid == 0) {
        // err was cleared before this kernel; every kv head ORs in its bits
        const uint32_t e = (bad_ctx ? ETI_ERRF_BAD_CTX : 0u) | (bad_page ? ETI_ERRF_BAD_PAGE : 0u) |
                           (timed_out ? ETI_ERRF_TIMEOUT : 0u) |
                           (timed_out && (flags & 4u) ? ETI_ERRF_DRAIN : 0u);
        if (e) atomicOr(a.err + b, e);
    }
    const int n = (bad_ctx || bad_page || timed_out) ? 0 : nb;
    const int e1 = min(j1, n);                   // the warp's blocks that count

    // B: Z - 1 = (sum c l1 + sum over the blocks below M of c) + (#blocks at
    // M - 1): log Z = log1p(Z - 1) keeps its relative precision when one
    // token takes nearly all of the attention
    float4 zs = make_float4(0.f, 0.f, 0.f, 0.f);  // (Z - 1 less the count, #at M, A, U)
    for (int j = j0 + jr; j < e1; j += BR)
        if (hv) {
            float4 s = sm[j * G + h];
            const bool top = !(s.x < M);
            const float c = top ? 1.f : exp_le0(s.x - M);
            zs.x += c * s.y + (top ? 0.f : c);
            zs.y += top ? 1.f : 0.f;
            const float z = c * (1.f + s.y);
            const float cu = c * (a.score_mode == 1 ? s.w : s.z);
            zs.z = fmaf(z, M - s.x, zs.z);
            zs.w += cu;
            s.y = z;
            s.z = cu;
            sm[j * G + h] = s;
        }
#pragma unroll
    for (int o = GP; o < 32; o <<= 1) {
        zs.x += __shfl_xor_sync(kAll, zs.x, o);
        zs.y += __shfl_xor_sync(kAll, zs.y, o);
        zs.z += __shfl_xor_sync(kAll, zs.z, o);
        zs.w += __shfl_xor_sync(kAll, zs.w, o);
    }
    if (lane < GP) red_s[wid][lane] = zs;
    __syncthreads();
    zs = red_s[0][h];
#pragma unroll
    for (int u = 1; u < NW; ++u) {
        const float4 v = red_s[u][h];
        zs.x += v.x; zs.y += v.y; zs.z += v.z; zs.w += v.w;
    }
    const float zm1 = zs.x + (zs.y - 1.f);
    const float lZ = log1pf(zm1), iZ = 1.f / (1.f + zm1);
    // H = sum_b I_b: log Z + (A - U) / Z (A); U / Z (E: stored surprisal); 1 (M)
    const float H = a.score_mode == 1 ? zs.w * iZ : a.score_mode == 2 ? 1.f : lZ + (zs.z - zs.w) * iZ;
    const float nH = H > 0.f ? (float)n / H : 0.f;

    // C: group scores (the GP lanes of a block agree), the threshold's kept
    // count, the argmax block
    const int kb = min(max(a.B_min, 0), n);
    float bs = -kInf;
    int bj = 0x7fffffff, kc = 0;
    for (int jb = j0; jb < e1; jb += BR) {       // the same trip count in every lane
        const int j = jb + jr;
        float s = -kInf;
        if (hv && j < e1) {
            const float4 v = sm[j * G + h];
            const float t = a.score_mode == 1 ? v.z * iZ
                          : a.score_mode == 2 ? v.y * iZ
                                              : fmaf(v.y, lZ + M - v.x, -v.z) * iZ;
            s = H > 0.f ? t * nH : 1.f;
        }
#pragma unroll
        for (int o = 1; o < GP; o <<= 1) s = fmaxf(s, __shfl_xor_sync(kAll, s, o));
        if (j < e1) {
            if (h == 0) {
                sc[j] = s;
                if (a.block_score) a.block_score[segbase + j] = s;
            }
            if (s > bs || bj == 0x7fffffff) { bs = s; bj = j; }
        }
        kc += __popc(__ballot_sync(kAll, h == 0 && j < e1 && (s >= th || kb >= n)));
    }
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const float ov = __shfl_xor_sync(kAll, bs, o);
        const int oj = __shfl_xor_sync(kAll, bj, o);
        if (ov > bs || (ov == bs && oj < bj)) { bs = ov; bj = oj; }
    }
    if (lane == 0) { arg_v[wid] = bs; arg_j[wid] = bj; cnt[wid] = kc; }
    __syncthreads();
    bs = arg_v[0];
    bj = arg_j[0];
    int off = 0, total = 0;
#pragma unroll
    for (int u = 0; u < NW; ++u) {
        if (u > 0 && (arg_v[u] > bs || (arg_v[u] == bs && arg_j[u] < bj))) { bs = arg_v[u]; bj = arg_j[u]; }
        off += u < wid ? cnt[u] : 0;
        total += cnt[u];
    }
    // the B_min = 1 budget's block joins the threshold's when it was left out
    const bool add = kb == 1 && n > 1 && !(bs >= th);
    const uint32_t below = (1u << lane) - 1u;

    if (!(kb > 1 && kb < n)) {
        // D: keep decisions and compaction of the warp's blocks, in order
        total += add ? 1 : 0;
        int run = off;
        for (int jb = j0; jb < e1; jb += 32) {
            const int j = jb + lane;
            const bool in = j < e1;
            const bool kt = in && (sc[j] >= th || kb >= n);
            const uint32_t bk = __ballot_sync(kAll, kt);
            const bool keep = kt || (add && j == bj);
            if (keep) a.kept_idx[segbase + run + __popc(bk & below) + (add && bj < j ? 1 : 0)] = j;
            if (in) {
                kf[j] = keep ? 1 : 0;
                if (a.keep_mask) a.keep_mask[segbase + j] = keep ? 1 : 0;
            }
            run += __popc(bk);
        }
        __syncwarp();                            // the keep flags of the warp's blocks
    } else {
        // the B_min budget: warp 0 takes the kb-th largest score key (ties: the
        // lowest indices) by a radix select, then ranks every block in order
        if (wid == 0) {
            uint32_t prefix = 0, mask = 0;
            int need = kb;
            for (int digit = 3; digit >= 0; --digit) {
                const int sh = digit * 8;
                for (int i = lane; i < 256; i += 32) hist[i] = 0;
                __syncwarp();
                for (int jb = 0; jb < n; jb += 32) {  // the same trip count in every lane
                    const int j = jb + lane;
                    const uint32_t key = j < n ? order_key(sc[j]) : 0u;
                    warp_hist_add(hist, (key >> sh) & 255, j < n && (key & mask) == prefix);
                }
                __syncwarp();
                // the bucket where the count from the top reaches `need`
                int cnt8[8], s8 = 0;
#pragma unroll
                for (int e = 0; e < 8; ++e) { cnt8[e] = hist[255 - (lane * 8 + e)]; s8 += cnt8[e]; }
                int incl = s8;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const int y = __shfl_up_sync(kAll, incl, o);
                    if (lane >= o) incl += y;
                }
                int above = incl - s8, dsel = -1, rsel = 0;
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    if (above < need && need <= above + cnt8[e]) {
                        dsel = 255 - (lane * 8 + e);
                        rsel = need - above;
                    }
                    above += cnt8[e];
                }
                const int src = __ffs(__ballot_sync(kAll, dsel >= 0)) - 1;
                dsel = __shfl_sync(kAll, dsel, src);
                rsel = __shfl_sync(kAll, rsel, src);
                prefix |= (uint32_t)dsel << sh;
                mask |= 255u << sh;
                need = rsel;
                __syncwarp();                    // before the histogram is cleared again
            }
            int run = 0, eq_run = 0;
            for (int jb = 0; jb < n; jb += 32) {
                const int j = jb + lane;
                const bool in = j < n;
                const float s = in ? sc[j] : -kInf;
                const uint32_t key = order_key(s);
                const bool eq = in && key == prefix;
                const uint32_t be = __ballot_sync(kAll, eq);
                const bool keep = in && (s >= th || key > prefix || (eq && eq_run + __popc(be & below) < need));
                eq_run += __popc(be);
                const uint32_t bk = __ballot_sync(kAll, keep);
                if (keep) a.kept_idx[segbase + run + __popc(bk & below)] = j;
                if (in) {
                    kf[j] = keep ? 1 : 0;
                    if (a.keep_mask) a.keep_mask[segbase + j] = keep ? 1 : 0;
                }
                run += __popc(bk);
            }
            if (lane == 0) sel[0] = run;
        }
        __syncthreads();
        total = sel[0];
    }
    for (int i = total + tid; i < a.max_blocks; i += NT) a.kept_idx[segbase + i] = -1;
    for (int j = n + tid; j < a.max_blocks; j += NT) {
        if (a.keep_mask) a.keep_mask[segbase + j] = 0;
        if (a.block_score) a.block_score[segbase + j] = 0.f;
    }
    if (tid == 0) a.kept_cnt[seg] = total;

    // E: softmax normaliser over the kept tokens of each head, (M_k, sum over
    // the kept blocks of (1 + l1_b) e^{m_b - M_k}): the z_b sums against M,
    // or, when the block holding a head's largest logit was left out, the
    // sums again against M_k from the stats (rare)
    if (a.kept_norm) {
        float mk = -kInf, lk = 0.f;
        for (int j = j0 + jr; j < e1; j += BR)
            if (hv && kf[j]) {
                const float4 v = sm[j * G + h];
                mk = fmaxf(mk, v.x);
                lk += v.y;
            }
#pragma unroll
        for (int o = GP; o < 32; o <<= 1) {
            mk = fmaxf(mk, __shfl_xor_sync(kAll, mk, o));
            lk += __shfl_xor_sync(kAll, lk, o);
        }
        if (lane < GP) { kn_m[wid][lane] = mk; kn_l[wid][lane] = lk; }
        __syncthreads();
        mk = -kInf;
        lk = 0.f;
#pragma unroll
        for (int u = 0; u < NW; ++u) { mk = fmaxf(mk, kn_m[u][h]); lk += kn_l[u][h]; }
        if (__syncthreads_or(hv && mk > -kInf && mk != M)) {
            float s2 = 0.f;
            for (int j = j0 + jr; j < e1; j += BR)
                if (hv && kf[j]) {
                    const float4 v = st[j * G + h];
                    s2 += (1.f + v.y) * exp_le0(v.x - mk);
                }
#pragma unroll
            for (int o = GP; o < 32; o <<= 1) s2 += __shfl_xor_sync(kAll, s2, o);
            if (lane < GP) kn_l[wid][lane] = s2;
            __syncthreads();
            lk = 0.f;
#pragma unroll
            for (int u = 0; u < NW; ++u) lk += kn_l[u][h];
        }
        if (tid < GP && hv) {
            float* kn = a.kept_norm + ((long long)b * a.Hq + kvh * a.g + h) * 2;
            kn[0] = mk;
            kn[1] = lk;
        }
    }
}

}  // namespace eti

using namespace eti;

// Whether the tile kernel takes segments of this shape (rule mode only).
bool eti_prune_tile_fits(int max_blocks, int g) { return (long long)max_blocks * g <= kTileItems; }

// Four warps a segment up to 4096 block-heads (fewer leave the longest
// segments' chains exposed, more add per-warp work: on the Llama-3-8B-shaped
// step 2/4/8/16 warps took 18.9/16.0/16.4/21.1 us), eight above.
cudaError_t eti_launch_prune_tile(const FinArgs& a, cudaStream_t stream) {
    const size_t smem = tile_smem(a.max_blocks, a.g);
    const int nw = (long long)a.max_blocks * a.g <= 4096 ? 4 : 8;
    const dim3 grid(a.B, a.Hkv);
#define ETI_TILE_NW(GG, NW)                                                                \
    if (nw == NW) {                                                                        \
        auto k = prune_finalize_tile_kernel<GG, NW>;                                       \
        cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem); \
        if (e != cudaSuccess) return e;                                                    \
        return eti_launch_pdl(k, grid, dim3(NW * 32), smem, stream, a);                    \
    }
#define ETI_TILE_CASE(GG)                                                                  \
    case GG: {                                                                             \
        ETI_TILE_NW(GG, 4)                                                                 \
        ETI_TILE_NW(GG, 8)                                                                 \
        return cudaErrorInvalidValue;                                                      \
    }
    switch (a.g) {
        ETI_TILE_CASE(1)
        ETI_TILE_CASE(2)
        ETI_TILE_CASE(3)
        ETI_TILE_CASE(4)
        ETI_TILE_CASE(5)
        ETI_TILE_CASE(6)
        ETI_TILE_CASE(7)
        ETI_TILE_CASE(8)
        default: return cudaErrorInvalidValue;
    }
#undef ETI_TILE_CASE
#undef ETI_TILE_NW
}
