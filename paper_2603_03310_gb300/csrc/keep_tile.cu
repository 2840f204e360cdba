// keep_tile.cu -- the keep set of segments whose block stats fit in shared
// memory (Section 3.2: the block entropy terms I_b, the block scores, the
// threshold / budget rule, compaction, the softmax normaliser over the kept
// tokens): one CTA of NW warps per (sequence, kv head) segment up to
// kTileItems block-heads, and for longer segments with B_min <= 1 a cluster
// of CL CTAs per segment, each staging its part.
//
// Warp w of CTA rank r owns a contiguous range of the segment's blocks: it
// stages their block stats (g float4 a block) in its CTA's shared memory with
// cp.async and takes, in rounds, query head h = l % GP of the blocks
// l / GP + k (32 / GP) of its range (lane l, GP the power of two >= g).
// Per-head sums are shuffle butterflies over the lanes of equal head, then
// NW partials in shared memory, then (a cluster) the CL CTAs' parts read
// through distributed shared memory, every CTA combining them in rank order
// so that all hold the same bits; the kept blocks are ranked by ballots in
// ascending block order within a warp and offset by the counts of the warps
// and ranks before it.  The work follows the segment's length (not
// max_blocks); three barriers (cluster barriers on a cluster) separate the
// passes over the staged stats:
//   A  the head's max M = max_b m_b (and the timeout marks of the scorer);
//   B  c_b = e^{m_b - M}, z_b = c_b (1 + l1_b); the sums Z - 1, A = sum z_b
//      (M - m_b) and U = sum c_b u_b give H = log Z + (A - U) / Z, the sum of
//      the block terms; (z_b, c_b u_b) replace (l1_b, u_b) in shared memory;
//   C  I_b = [z_b (log Z + M - m_b) - c_b u_b] / Z, the group score (the
//      largest n_b I_b / H over the heads of the block), the threshold's
//      kept count and the argmax block of each warp;
//   D  keep decisions and compaction (the B_min > 1 budget, one CTA only: a
//      radix select of the kb-th score key by warp 0, which then ranks every
//      block);
//   E  (M_k, L_k) of each head over the kept blocks: the z_b sums against M,
//      taken again against M_k from the stats when the block holding a
//      head's largest logit was left out.
#include "keep_set.cuh"

namespace eti {

constexpr int kTileItems = 8192;        // largest max_blocks * g one CTA stages
constexpr int kTileClusterItems = 32768; // largest max_blocks * g a cluster of up to 8 CTAs stages
constexpr int kTileCtaItems = 4096;     // block-heads a CTA of a cluster stages at most

// The same 16 bytes of shared memory of every CTA rank of the cluster, all the
// loads issued before any is used (each is a round trip to another SM).
template <int CL>
__device__ __forceinline__ void ld_ranks_f32x4(float4 (&v)[CL], const float4* p) {
    const uint32_t a = smem_u32(p);
#pragma unroll
    for (int r = 0; r < CL; ++r) {
        uint32_t ra;
        asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(ra) : "r"(a), "r"(r));
        asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
                     : "=f"(v[r].x), "=f"(v[r].y), "=f"(v[r].z), "=f"(v[r].w) : "r"(ra) : "memory");
    }
}

// Blocks of the segment that CTA rank cr of CL stages, at most: whole rounds
// of 32 / GP blocks for each of its NW warps.
__host__ __device__ inline int tile_cap_blocks(int max_blocks, int NW, int CL, int BR) {
    const int per_warp = ((max_blocks + CL * NW - 1) / (CL * NW) + BR - 1) / BR * BR;
    return per_warp * NW;
}

// shared memory of a CTA: the radix histogram, the stats of its blocks, their
// scores, their keep flags
inline size_t tile_smem(int cap_blocks, int g) {
    return (1024 + (size_t)cap_blocks * g * 16 + (size_t)cap_blocks * 5 + 15) / 16 * 16;
}

template <int G, int NW, int CL>
__global__ void __launch_bounds__(NW * 32) prune_finalize_tile_kernel(const FinArgs a) {
    constexpr int GP = FlatGP<G>::v;
    constexpr int BR = 32 / GP;                  // blocks of a round
    constexpr int NT = NW * 32;
    constexpr unsigned kAll = 0xffffffffu;
    pdl_trigger();
    pdl_wait();
    const int capb = tile_cap_blocks(a.max_blocks, NW, CL, BR);
    extern __shared__ __align__(16) unsigned char tile_smem_raw[];
    int* hist = reinterpret_cast<int*>(tile_smem_raw);
    float4* sm = reinterpret_cast<float4*>(tile_smem_raw + 1024);
    float* sc = reinterpret_cast<float*>(tile_smem_raw + 1024 + (size_t)capb * G * 16);
    uint8_t* kf = reinterpret_cast<uint8_t*>(sc + capb);
    __shared__ float red_m[NW][GP];
    __shared__ float4 red_s[NW][GP];
    __shared__ unsigned red_f[NW];
    __shared__ float arg_v[NW];
    __shared__ int arg_j[NW], cnt[NW];
    __shared__ float kn_m[NW][GP], kn_l[NW][GP];
    __shared__ int sel[2];
    // cluster exchange slots (one per exchange, never reused): the CTA's part
    __shared__ float4 x1[GP], x2[GP], x4[GP], x5[GP];   // per head
    __shared__ float4 x3;                                // argmax value, block, kept count
    // grid (B * CL, Hkv), clusters of CL CTAs along x: one cluster a segment
    const int cr = CL > 1 ? (int)cluster_rank() : 0;
    const int b = blockIdx.x / CL, kvh = blockIdx.y;
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
    // warp w of CTA rank cr owns blocks [j0, j1): contiguous ranges in block
    // order, whole rounds; the CTA's blocks start at cb0 (local index j - cb0)
    const int q = ((nb + CL * NW - 1) / (CL * NW) + BR - 1) / BR * BR;
    const int cb0 = min(nb, cr * NW * q);
    const int j0 = min(nb, (cr * NW + wid) * q), j1 = min(nb, j0 + q);

    // stage the warp's stats; check its page ids meanwhile
    const uint32_t sbase = smem_u32(sm);
    for (int i = j0 * G + lane; i < j1 * G; i += 32) cp_async_16(sbase + (i - cb0 * G) * 16, st + i, true);
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
            const float4 s = sm[(j - cb0) * G + h];
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
    if constexpr (CL > 1) {
        // the cluster's: every CTA combines the ranks' parts in rank order
        if (tid < GP) x1[tid] = make_float4(M, __uint_as_float(flags), 0.f, 0.f);
        cluster_sync();
        float4 v[CL];
        ld_ranks_f32x4<CL>(v, &x1[h]);
        M = -kInf;
        flags = 0;
#pragma unroll
        for (int p = 0; p < CL; ++p) { M = fmaxf(M, v[p].x); flags |= __float_as_uint(v[p].y); }
    }
    const bool bad_page = (flags & 1u) != 0;
    const bool timed_out = (flags & 2u) && !bad_page;
    if (a.err && tid == 0 && cr == 0) {
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
            float4 s = sm[(j - cb0) * G + h];
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
            sm[(j - cb0) * G + h] = s;
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
    if constexpr (CL > 1) {
        if (tid < GP) x2[tid] = zs;
        cluster_sync();
        float4 v[CL];
        ld_ranks_f32x4<CL>(v, &x2[h]);
        zs = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int p = 0; p < CL; ++p) { zs.x += v[p].x; zs.y += v[p].y; zs.z += v[p].z; zs.w += v[p].w; }
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
            const float4 v = sm[(j - cb0) * G + h];
            const float t = a.score_mode == 1 ? v.z * iZ
                          : a.score_mode == 2 ? v.y * iZ
                                              : fmaf(v.y, lZ + M - v.x, -v.z) * iZ;
            s = H > 0.f ? t * nH : 1.f;
        }
#pragma unroll
        for (int o = 1; o < GP; o <<= 1) s = fmaxf(s, __shfl_xor_sync(kAll, s, o));
        if (j < e1) {
            if (h == 0) {
                sc[j - cb0] = s;
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
    if constexpr (CL > 1) {
        // the cluster's argmax; the kept counts of the lower ranks offset ours
        if (tid == 0) x3 = make_float4(bs, __int_as_float(bj), __int_as_float(total), 0.f);
        cluster_sync();
        float4 v[CL];
        ld_ranks_f32x4<CL>(v, &x3);
        bs = -kInf;
        bj = 0x7fffffff;
        total = 0;
#pragma unroll
        for (int p = 0; p < CL; ++p) {
            const float ov = v[p].x;
            const int oj = __float_as_int(v[p].y), oc = __float_as_int(v[p].z);
            if (ov > bs || (ov == bs && oj < bj)) { bs = ov; bj = oj; }
            off += p < cr ? oc : 0;
            total += oc;
        }
    }
    // the B_min = 1 budget's block joins the threshold's when it was left out
    const bool add = kb == 1 && n > 1 && !(bs >= th);
    const uint32_t below = (1u << lane) - 1u;

    // (a cluster takes segments only for B_min <= 1: no radix select there)
    if (CL > 1 || !(kb > 1 && kb < n)) {
        // D: keep decisions and compaction of the warp's blocks, in order
        total += add ? 1 : 0;
        int run = off;
        for (int jb = j0; jb < e1; jb += 32) {
            const int j = jb + lane;
            const bool in = j < e1;
            const bool kt = in && (sc[j - cb0] >= th || kb >= n);
            const uint32_t bk = __ballot_sync(kAll, kt);
            const bool keep = kt || (add && j == bj);
            if (keep) a.kept_idx[segbase + run + __popc(bk & below) + (add && bj < j ? 1 : 0)] = j;
            if (in) {
                kf[j - cb0] = keep ? 1 : 0;
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
    for (int i = total + cr * NT + tid; i < a.max_blocks; i += CL * NT) a.kept_idx[segbase + i] = -1;
    for (int j = n + cr * NT + tid; j < a.max_blocks; j += CL * NT) {
        if (a.keep_mask) a.keep_mask[segbase + j] = 0;
        if (a.block_score) a.block_score[segbase + j] = 0.f;
    }
    if (tid == 0 && cr == 0) a.kept_cnt[seg] = total;

    // E: softmax normaliser over the kept tokens of each head, (M_k, sum over
    // the kept blocks of (1 + l1_b) e^{m_b - M_k}): the z_b sums against M,
    // or, when the block holding a head's largest logit was left out, the
    // sums again against M_k from the stats (rare)
    if (a.kept_norm) {
        float mk = -kInf, lk = 0.f;
        for (int j = j0 + jr; j < e1; j += BR)
            if (hv && kf[j - cb0]) {
                const float4 v = sm[(j - cb0) * G + h];
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
        if constexpr (CL > 1) {
            if (tid < GP) x4[tid] = make_float4(mk, lk, 0.f, 0.f);
            cluster_sync();
            float4 v[CL];
            ld_ranks_f32x4<CL>(v, &x4[h]);
            mk = -kInf;
            lk = 0.f;
#pragma unroll
            for (int p = 0; p < CL; ++p) { mk = fmaxf(mk, v[p].x); lk += v[p].y; }
        }
        // the same decision in every thread of every CTA of the cluster
        if (__syncthreads_or(hv && mk > -kInf && mk != M)) {
            float s2 = 0.f;
            for (int j = j0 + jr; j < e1; j += BR)
                if (hv && kf[j - cb0]) {
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
            if constexpr (CL > 1) {
                if (tid < GP) x5[tid] = make_float4(lk, 0.f, 0.f, 0.f);
                cluster_sync();
                float4 v[CL];
                ld_ranks_f32x4<CL>(v, &x5[h]);
                lk = 0.f;
#pragma unroll
                for (int p = 0; p < CL; ++p) lk += v[p].x;
            }
        }
        if (tid < GP && hv && cr == 0) {
            float* kn = a.kept_norm + ((long long)b * a.Hq + kvh * a.g + h) * 2;
            kn[0] = mk;
            kn[1] = lk;
        }
    }
    // no CTA of the cluster leaves while another may still read its shared memory
    if constexpr (CL > 1) cluster_sync();
}

}  // namespace eti

using namespace eti;

// CTAs of a segment's cluster for this shape (1: one CTA, no cluster).
static int tile_cluster(long long items) { return items <= kTileItems ? 1 : items <= 4 * kTileCtaItems ? 4 : 8; }

// Whether the tile kernel takes segments of this shape in the rule mode:
// up to 8192 block-heads; up to 32768 with B_min <= 1 (no radix select on a
// cluster) when the clusters of all `segs` segments run in about one wave
// (four CTAs an SM).  Many long segments run faster on the segment kernel:
// on 1024 segments of up to 2048 blocks x 8 heads (9 waves of 4-CTA
// clusters) 121 us against its 91 us, where 64 segments of up to 8192
// blocks x 4 heads took 33 us against the wide kernel's 47 us.
bool eti_prune_tile_fits(int max_blocks, int g, int B_min, int segs, int sms) {
    const long long items = (long long)max_blocks * g;
    if (items <= kTileItems) return true;
    return B_min <= 1 && items <= kTileClusterItems && (long long)segs * tile_cluster(items) <= 4LL * sms;
}

template <int G, int NW, int CL>
static cudaError_t launch_tile(const FinArgs& a, cudaStream_t stream) {
    constexpr int BR = 32 / FlatGP<G>::v;
    const size_t smem = tile_smem(tile_cap_blocks(a.max_blocks, NW, CL, BR), G);
    auto k = prune_finalize_tile_kernel<G, NW, CL>;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(a.B * CL, a.Hkv);
    cfg.blockDim = dim3(NW * 32);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = CL;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = CL > 1 ? 2 : 1;
    return cudaLaunchKernelEx(&cfg, k, a);
}

template <int G>
static cudaError_t launch_tile_shape(const FinArgs& a, cudaStream_t stream) {
    const long long items = (long long)a.max_blocks * G;
    if (items <= 4096) return launch_tile<G, 4, 1>(a, stream);
    if (items <= kTileItems) return launch_tile<G, 8, 1>(a, stream);
    // a cluster of four or eight CTAs of eight warps, each staging up to
    // 4096 block-heads
    if (tile_cluster(items) == 4) return launch_tile<G, 8, 4>(a, stream);
    return launch_tile<G, 8, 8>(a, stream);
}

// Four warps a CTA up to 4096 block-heads (fewer leave the longest
// segments' chains exposed, more add per-warp work: on the Llama-3-8B-shaped
// step 2/4/8/16 warps took 18.9/16.0/16.4/21.1 us), eight above, and above
// 8192 a cluster of CTAs a segment.  The caller sends only the shapes that
// eti_prune_tile_fits accepts; a cluster launch the device refuses returns
// its error, and the caller falls back to the wide kernel.
cudaError_t eti_launch_prune_tile(const FinArgs& a, cudaStream_t stream) {
    switch (a.g) {
        case 1: return launch_tile_shape<1>(a, stream);
        case 2: return launch_tile_shape<2>(a, stream);
        case 3: return launch_tile_shape<3>(a, stream);
        case 4: return launch_tile_shape<4>(a, stream);
        case 5: return launch_tile_shape<5>(a, stream);
        case 6: return launch_tile_shape<6>(a, stream);
        case 7: return launch_tile_shape<7>(a, stream);
        case 8: return launch_tile_shape<8>(a, stream);
        default: return cudaErrorInvalidValue;
    }
}
