// prune_wide.cu -- the keep-set kernels for segments longer than the tile
// kernel stages (more than 8192 block-heads), and for the given keep sets of
// a standalone decode (Section 3.2).
#include "keep_set.cuh"

namespace eti {

// ---------------------------------------------------------------------------
// prune_finalize for segments of any size (and for the given keep sets), in
// a flat layout: thread t owns query head h = t % GP of the blocks
// r * RB + t / GP + k * JS, k < kFlatPer, in rounds r of RB = JS * kFlatPer
// blocks.  Every pass walks the rounds and re-reads the block stats
// (L2-resident after the first pass), so loads are coalesced and nothing of
// size max_blocks lives in registers; the group scores, then the keep flags,
// live in shared memory ([max_blocks] floats); with kTerm the term of every
// block-head too.  Ranks in ascending block order (budget ties, compaction)
// are ballot scans per round with a running base.
//
// A segment is handled by a cluster of kCl CTAs (kCl = 1: one CTA): CTA rank
// c takes a contiguous run of the rounds.  The per-head reductions, the error
// flags, the budget histograms and argmax, and the counts that offset the
// ordered ranks are exchanged through distributed shared memory, each CTA
// combining all ranks' values in rank order, so every CTA of the cluster
// holds the same bits.  Cluster barriers sit in code every CTA of the cluster
// runs the same number of times (it depends on the segment only).
constexpr int kWideX = 16;    // exchange slots (one per exchange, never reused)

template <int G, int NT, bool kTerm, int kCl>
__global__ void __launch_bounds__(NT, NT >= 1024 ? 1 : 2)
prune_finalize_wide_kernel(const FinArgs a) {
    constexpr int GP = FlatGP<G>::v;
    constexpr int JS = NT / GP;                  // block stride between a thread's chunks
    constexpr int RB = JS * kFlatPer;            // blocks per round
    pdl_trigger();
    pdl_wait();
    extern __shared__ __align__(16) float wf_smem[];
    float* sh = wf_smem;                         // [max_blocks]: group scores, then keep flags
    // kTerm: [max_blocks * GP] per block-head e^{m_b - M}, then the term I_b
    // (index j * GP + h: a warp's accesses are consecutive); with
    // a.share_cache also [max_blocks * GP] shares (1 + l1_b) e^{m_b - M} of Z,
    // which give the kept-token normaliser when the head's top block is kept
    float* sh_t = wf_smem + a.max_blocks;
    float* sh_s = sh_t + (size_t)a.max_blocks * GP;
    const bool share = kTerm && a.share_cache;
    __shared__ float red[4][2 * 32 * GP];
    __shared__ float fin[2][2 * GP];             // two-stage reductions: the final per-head values
    __shared__ int scan[2][kFlatPer * 32 + 1];
    __shared__ int hist[2][256];
    __shared__ int hsum[256];
    __shared__ int sel_digit, sel_rem;
    __shared__ float arg_v[32];
    __shared__ int arg_j[32];
    __shared__ float xf[kWideX][2 * GP];         // exchanged per-head values
    __shared__ int xi[kWideX][2];                // exchanged integers
    __shared__ int isum[NT / 32];
    const int cr = kCl > 1 ? (int)cluster_rank() : 0;
    const int seg = blockIdx.x / kCl;
    const int b = seg / a.Hkv, kvh = seg - b * a.Hkv;
    const int tid = threadIdx.x, lane = tid & 31;
    const int h = lane & (GP - 1);
    const int jt = tid / GP;
    const int L = a.ctx_lens[b];
    const bool bad_ctx = L < 0 || L > a.max_blocks * a.P;
    const int nb = bad_ctx ? 0 : (L + a.P - 1) / a.P;
    const int nr = (nb + RB - 1) / RB;           // rounds of the segment
    const int rsplit = (nr + kCl - 1) / kCl;
    const int r_lo = min(nr, cr * rsplit), r_hi = min(nr, r_lo + rsplit);   // this CTA's rounds
    const long long segbase = (long long)seg * a.max_blocks;
    const float4* st = a.stats + segbase * G;
    auto stat = [&](int j) {
        float4 v = st[(long long)j * G + h];
        if (a.score_mode == 1) v.z = v.w;        // .z: u (mode A) or sum e^{x-m} s_i (mode E)
        return v;
    };
    int xslot = 0;
    // sum of one int per thread over the CTA
    auto block_sum = [&](int v) {
        v = warp_sum_i(v);
        if (lane == 0) isum[tid >> 5] = v;
        __syncthreads();
        int t = 0;
        for (int u = 0; u < NT / 32; ++u) t += isum[u];
        __syncthreads();
        return t;
    };
    // per-head values (head h in every thread): combined over the cluster
    auto cl_heads = [&](float* v, int N, bool is_max) {
        if (kCl == 1) return;
        float* x = xf[xslot++];
        if (tid < GP)
            for (int i = 0; i < N; ++i) x[i * GP + tid] = v[i];
        cluster_sync();
        for (int i = 0; i < N; ++i) {
            float r = ld_cluster_f32(&x[i * GP + h], 0);
            for (int p = 1; p < kCl; ++p) {
                const float y = ld_cluster_f32(&x[i * GP + h], (uint32_t)p);
                r = is_max ? fmaxf(r, y) : r + y;
            }
            v[i] = r;
        }
    };
    // one integer per CTA: returns the sum over the cluster and, in *below,
    // the sum over the lower ranks
    auto cl_count = [&](int v, int* below) {
        if (kCl == 1) { *below = 0; return v; }
        int* x = xi[xslot++];
        if (tid == 0) x[0] = v;
        cluster_sync();
        int tot = 0, lo = 0;
        for (int p = 0; p < kCl; ++p) {
            const int y = ld_cluster_s32(x, (uint32_t)p);
            if (p < cr) lo += y;
            tot += y;
        }
        *below = lo;
        return tot;
    };

    // page ids of the segment's blocks (split over the cluster), stale stats,
    // the per-head max
    const int bad = any_bad_page(a.block_table + (long long)b * a.max_blocks, cr * NT + tid, kCl * NT, nb,
                                 a.num_pages);
    int stale = 0;
    float Mh[1] = {-kInf};
    for (int r = r_lo; r < r_hi; ++r)
#pragma unroll
        for (int k = 0; k < kFlatPer; ++k) {
            const int j = r * RB + jt + k * JS;
            if (h < G && j < nb) {
                const float x = st[(long long)j * G + h].x;
                stale |= (x != x);               // NaN max: the scoring pass gave up on this block
                Mh[0] = fmaxf(Mh[0], x);
            }
        }
    int dummy;
    const bool bad_page = cl_count(__syncthreads_or(bad) != 0, &dummy) != 0;
    const bool timed_out = cl_count(__syncthreads_or(stale) != 0, &dummy) != 0 && !bad_page;
    bool drain = false;
    if (timed_out) {
        // rare: a block marked l - 1 = +inf had a copy in flight when the drain gave up
        int d = 0;
        for (int r = r_lo; r < r_hi; ++r)
#pragma unroll
            for (int k = 0; k < kFlatPer; ++k) {
                const int j = r * RB + jt + k * JS;
                if (h < G && j < nb) {
                    const float4 s4 = st[(long long)j * G + h];
                    d |= (s4.x != s4.x) && s4.y == kInf;
                }
            }
        drain = cl_count(__syncthreads_or(d) != 0, &dummy) != 0;
    }
    if (a.err && tid == 0 && cr == 0) {
        // err was cleared before this kernel; every kv head ORs in its bits
        const uint32_t e = (bad_ctx ? ETI_ERRF_BAD_CTX : 0u) | (bad_page ? ETI_ERRF_BAD_PAGE : 0u) |
                           (timed_out ? ETI_ERRF_TIMEOUT : 0u) | (drain ? ETI_ERRF_DRAIN : 0u);
        if (e) atomicOr(a.err + b, e);
    }
    const int n = (bad_ctx || bad_page || timed_out) ? 0 : nb;
    float M = -kInf;
    if (n > 0) {
        head_reduce2<GP, 1, true>(Mh, red[0], fin[1 - 1]);
        cl_heads(Mh, 1, true);
        M = Mh[0];
    }

    const int jlo = r_lo * RB, jhi = min(n, r_hi * RB);   // this CTA's blocks of the segment
    int kbase = 0;                               // kept blocks listed so far (one-CTA rule mode)
    if (!a.given) {
        if (n > 0) {
            // Z - 1 = sum_b c_b l1_b + sum_{b: m_b < M} c_b + (#blocks at M - 1),
            // c_b = e^{m_b - M} (the blocks at the max are counted, not summed)
            float zs[2] = {0.f, 0.f};
            for (int r = r_lo; r < r_hi; ++r)
#pragma unroll
                for (int k = 0; k < kFlatPer; ++k) {
                    const int j = r * RB + jt + k * JS;
                    if (h < G && j < n) {
                        const float4 v = stat(j);
                        const bool top = !(v.x < M);
                        const float c = top ? 1.f : exp_le0(v.x - M);
                        zs[0] += c * v.y + (top ? 0.f : c);
                        zs[1] += top ? 1.f : 0.f;
                        if (kTerm) sh_t[j * GP + h] = c;
                        if (share) sh_s[j * GP + h] = (1.f + v.y) * c;
                    }
                }
            head_reduce2<GP, 2, false>(zs, red[1], fin[2 - 1]);
            cl_heads(zs, 2, false);
            const float zm1 = zs[0] + (zs[1] - 1.f);
            const float lZ = log1pf(zm1), iZ = 1.f / (1.f + zm1);
            // I_b = e^{m_b - M}[(1 + l1_b)(log Z + M - m_b) - u_b] / Z; H = sum_b I_b
            auto Ib = [&](float4 v, float c) {
                if (a.score_mode == 1) return c * v.z * iZ;                 // E
                if (a.score_mode == 2) return c * (1.f + v.y) * iZ;         // M
                return c * ((1.f + v.y) * (lZ + M - v.x) - v.z) * iZ;
            };
            float Hs[1] = {0.f};
            for (int r = r_lo; r < r_hi; ++r)
#pragma unroll
                for (int k = 0; k < kFlatPer; ++k) {
                    const int j = r * RB + jt + k * JS;
                    if (h < G && j < n) {
                        const float4 v = stat(j);
                        const float t = Ib(v, kTerm ? sh_t[j * GP + h] : (v.x < M ? exp_le0(v.x - M) : 1.f));
                        if (kTerm) sh_t[j * GP + h] = t;
                        Hs[0] += t;
                    }
                }
            head_reduce2<GP, 1, false>(Hs, red[2], fin[1 - 1]);
            cl_heads(Hs, 1, false);
            const float nH = Hs[0] > 0.f ? (float)n / Hs[0] : 0.f;
            // group score: the largest normalised term over the heads of the block
            for (int r = r_lo; r < r_hi; ++r)
#pragma unroll
                for (int k = 0; k < kFlatPer; ++k) {
                    const int j = r * RB + jt + k * JS;
                    float sc = -kInf;
                    if (h < G && j < n) {
                        float t;
                        if (kTerm) {
                            t = sh_t[j * GP + h];
                        } else {
                            const float4 v = stat(j);
                            t = Ib(v, v.x < M ? exp_le0(v.x - M) : 1.f);
                        }
                        sc = Hs[0] > 0.f ? t * nH : 1.f;
                    }
#pragma unroll
                    for (int o = 1; o < GP; o <<= 1) sc = fmaxf(sc, __shfl_xor_sync(0xffffffffu, sc, o));
                    if (h == 0 && j < n) sh[j] = sc;
                }
        }
        __syncthreads();
        if (a.block_score) {
            for (int j = jlo + tid; j < jhi; j += NT) a.block_score[segbase + j] = sh[j];
            for (int j = n + cr * NT + tid; j < a.max_blocks; j += kCl * NT) a.block_score[segbase + j] = 0.f;
        }

        // B_min budget: the first kb blocks by (score desc, index asc)
        const float th = a.theta ? a.theta[b] : kInf;
        const int kb = min(max(a.B_min, 0), n);
        int arg = -1;
        uint32_t kth = 0u;
        int need = 0;
        if (kb == 1 && n > 1) {
            float bs = -kInf;
            int bj = 0x7fffffff;
            for (int j = jlo + tid; j < jhi; j += NT) {
                const float v = sh[j];
                if (v > bs || bj == 0x7fffffff) { bs = v; bj = j; }
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                const float ov = __shfl_xor_sync(0xffffffffu, bs, o);
                const int oj = __shfl_xor_sync(0xffffffffu, bj, o);
                if (ov > bs || (ov == bs && oj < bj)) { bs = ov; bj = oj; }
            }
            if (lane == 0) { arg_v[tid >> 5] = bs; arg_j[tid >> 5] = bj; }
            __syncthreads();
            for (int u = 0; u < NT / 32; ++u)
                if (arg_v[u] > bs || (arg_v[u] == bs && arg_j[u] < bj)) { bs = arg_v[u]; bj = arg_j[u]; }
            if (kCl > 1) {
                const int s = xslot++;
                if (tid == 0) { xf[s][0] = bs; xi[s][0] = bj; }
                cluster_sync();
                bs = -kInf;
                bj = 0x7fffffff;
                for (int p = 0; p < kCl; ++p) {
                    const float ov = ld_cluster_f32(&xf[s][0], (uint32_t)p);
                    const int oj = ld_cluster_s32(&xi[s][0], (uint32_t)p);
                    if (oj != 0x7fffffff && (ov > bs || bj == 0x7fffffff || (ov == bs && oj < bj))) { bs = ov; bj = oj; }
                }
            }
            arg = bj;
        } else if (kb > 1 && kb < n) {
            uint32_t prefix = 0, mask = 0;
            need = kb;
            for (int digit = 3; digit >= 0; --digit) {
                const int shf = digit * 8;
                int* hd = hist[digit & 1];
                for (int i = tid; i < 256; i += NT) hd[i] = 0;
                __syncthreads();
                for (int j0 = jlo; j0 < jhi; j0 += NT) {  // the same trip count for every lane
                    const int j = j0 + tid;
                    const uint32_t key = j < jhi ? order_key(sh[j]) : 0u;
                    warp_hist_add(hd, (key >> shf) & 255, j < jhi && (key & mask) == prefix);
                }
                if (kCl > 1) {
                    cluster_sync();
                    for (int i = tid; i < 256; i += NT) {
                        int t = 0;
                        for (int p = 0; p < kCl; ++p) t += ld_cluster_s32(&hd[i], (uint32_t)p);
                        hsum[i] = t;
                    }
                } else {
                    __syncthreads();
                    for (int i = tid; i < 256; i += NT) hsum[i] = hd[i];
                }
                __syncthreads();
                // bucket where the count from the top reaches `need`
                if (tid < 32) {
                    int cnt8[8], s8 = 0;
#pragma unroll
                    for (int e = 0; e < 8; ++e) { cnt8[e] = hsum[255 - (tid * 8 + e)]; s8 += cnt8[e]; }
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
                prefix |= (uint32_t)sel_digit << shf;
                mask |= 255u << shf;
                need = sel_rem;
                __syncthreads();
            }
            kth = prefix;
        }
        // keep flags: threshold, budget (ties at the k-th key to the lower index:
        // this CTA's ties are ranked after those of the lower ranks)
        const bool sel = kb > 1 && kb < n;
        int eq_base = 0;
        if (sel) {
            int eq = 0;
            for (int j = jlo + tid; j < jhi; j += NT) eq += order_key(sh[j]) == kth;
            int below;
            cl_count(block_sum(eq), &below);
            eq_base = below;
        }
        for (int r = r_lo; r < r_hi; ++r) {
            bool eq[kFlatPer], keep[kFlatPer];
            int eq_pos[kFlatPer];
#pragma unroll
            for (int k = 0; k < kFlatPer; ++k) {
                const int j = r * RB + jt + k * JS;
                const float sc = j < n ? sh[j] : -kInf;
                const uint32_t key = order_key(sc);
                keep[k] = j < n && (sc >= th || kb >= n || j == arg || (sel && key > kth));
                eq[k] = sel && j < n && key == kth;
            }
            if (sel) {
                const int c = flat_ranks<GP>(eq, eq_pos, scan[r & 1]);
#pragma unroll
                for (int k = 0; k < kFlatPer; ++k) keep[k] |= eq[k] && eq_base + eq_pos[k] < need;
                eq_base += c;
            }
            if (kCl == 1) {
                // one CTA: the ranks of this round follow those of the rounds
                // before it, so the kept list is written here
                int pos[kFlatPer];
                const int c = flat_ranks<GP>(keep, pos, scan[(r + 1) & 1]);
#pragma unroll
                for (int k = 0; k < kFlatPer; ++k) {
                    const int j = r * RB + jt + k * JS;
                    if (h == 0 && keep[k]) a.kept_idx[segbase + kbase + pos[k]] = j;
                    if (a.keep_mask && h == 0 && j < n) a.keep_mask[segbase + j] = keep[k] ? 1 : 0;
                }
                kbase += c;
            }
            __syncthreads();    // every lane of a block has read its score
#pragma unroll
            for (int k = 0; k < kFlatPer; ++k) {
                const int j = r * RB + jt + k * JS;
                if (h == 0 && j < n) sh[j] = keep[k] ? 1.f : 0.f;
            }
        }
        __syncthreads();
    } else {
        // given keep set: a list, a mask, or every block (this CTA's blocks)
        if (a.given_idx) {
            for (int j = jlo + tid; j < jhi; j += NT) sh[j] = 0.f;
            __syncthreads();
            const int c = min(max(a.given_cnt[seg], 0), a.max_blocks);
            for (int i = tid; i < c; i += NT) {
                const int j = a.given_idx[segbase + i];
                if (j >= jlo && j < jhi) sh[j] = 1.f;
            }
        } else {
            for (int j = jlo + tid; j < jhi; j += NT)
                sh[j] = a.given_mask ? (a.given_mask[segbase + j] ? 1.f : 0.f) : 1.f;
        }
        __syncthreads();
    }

    // compaction (ascending block index), round by round, after the kept
    // blocks of the lower ranks (one-CTA rule mode: done with the flags)
    const bool listed = kCl == 1 && !a.given;
    int total = kbase, base = 0;
    if (!listed) {
        int cnt = 0;
        for (int j = jlo + tid; j < jhi; j += NT) cnt += sh[j] != 0.f;
        total = cl_count(block_sum(cnt), &base);
    }
    for (int r = listed ? r_hi : r_lo; r < r_hi; ++r) {
        bool keep[kFlatPer];
        int pos[kFlatPer];
#pragma unroll
        for (int k = 0; k < kFlatPer; ++k) {
            const int j = r * RB + jt + k * JS;
            keep[k] = j < n && sh[j] != 0.f;
        }
        const int c = flat_ranks<GP>(keep, pos, scan[r & 1]);
#pragma unroll
        for (int k = 0; k < kFlatPer; ++k) {
            const int j = r * RB + jt + k * JS;
            if (h == 0 && keep[k]) a.kept_idx[segbase + base + pos[k]] = j;
            if (a.keep_mask && h == 0 && j < n) a.keep_mask[segbase + j] = keep[k] ? 1 : 0;
        }
        base += c;
    }
    for (int i = total + cr * NT + tid; i < a.max_blocks; i += kCl * NT) a.kept_idx[segbase + i] = -1;
    if (a.keep_mask)
        for (int j = n + cr * NT + tid; j < a.max_blocks; j += kCl * NT) a.keep_mask[segbase + j] = 0;
    if (tid == 0 && cr == 0) a.kept_cnt[seg] = total;

    // softmax normaliser over the kept tokens of each query head
    if (a.kept_norm) {
        float Mk[1] = {-kInf};
        for (int r = r_lo; r < r_hi; ++r)
#pragma unroll
            for (int k = 0; k < kFlatPer; ++k) {
                const int j = r * RB + jt + k * JS;
                if (h < G && j < n && sh[j] != 0.f) Mk[0] = fmaxf(Mk[0], st[(long long)j * G + h].x);
            }
        head_reduce2<GP, 1, true>(Mk, red[3], fin[1 - 1]);
        cl_heads(Mk, 1, true);
        float Lk[1] = {0.f};
        // (the rule mode's M is the head's max over all blocks: when the top
        // block is kept the cached shares already have the right scale)
        const bool cached = share && !a.given && Mk[0] == M;
        for (int r = r_lo; r < r_hi; ++r)
#pragma unroll
            for (int k = 0; k < kFlatPer; ++k) {
                const int j = r * RB + jt + k * JS;
                if (h < G && j < n && sh[j] != 0.f) {
                    if (cached) {
                        Lk[0] += sh_s[j * GP + h];
                    } else {
                        const float4 v = st[(long long)j * G + h];
                        Lk[0] += (1.f + v.y) * exp_le0(v.x - Mk[0]);
                    }
                }
            }
        head_reduce2<GP, 1, false>(Lk, red[0], fin[1 - 1]);
        cl_heads(Lk, 1, false);
        if (tid < GP && h < G && cr == 0) {
            float* kn = a.kept_norm + ((long long)b * a.Hq + kvh * a.g + h) * 2;
            kn[0] = Mk[0];
            kn[1] = Lk[0];
        }
    }
    // no CTA of the cluster leaves while another may still read its shared memory
    if (kCl > 1) cluster_sync();
}

// ---------------------------------------------------------------------------
// prune_finalize_seg_kernel: the rule mode for a segment whose per-block-head
// terms fit in shared memory (max_blocks * (GP + 1) floats), one CTA of NT
// threads per (sequence, kv head) segment, two CTAs per SM.
//  - three passes over the block stats in the head-lane layout (thread t:
//    head t % GP of blocks t / GP, t / GP + NT / GP, ... up to the segment's
//    end, not to max_blocks): the per-head max, then e^{m_b - M} and Z, then
//    the terms I_b and H, the terms kept in shared memory; the first pass
//    reads the stats from HBM, the next two from L2.  (Folding the terms into
//    the second pass as pairs (A_b, B_b) with I_b = (A_b log Z + B_b) / Z
//    needs twice the shared memory, one CTA per SM, and was slower: 168
//    against 117 us on the 70B-shaped step);
//  - per block, over shared memory (thread t: the contiguous run of blocks
//    [t q, (t + 1) q)): the group score max_h n I_b^(h) / H^(h), the budget
//    (argmax, or a radix select with ties to the lower index), the keep
//    flag, and the compaction from an exclusive scan of the runs' counts;
//  - one pass over the kept blocks' stats for the kept-token normaliser
//    (an online max and sum per head).
template <int G, int NT>
__global__ void __launch_bounds__(NT, 2)
prune_finalize_seg_kernel(const FinArgs a) {
    constexpr int GP = FlatGP<G>::v;
    constexpr int JS = NT / GP;                  // block stride of a head lane
    constexpr int NW = NT / 32;
    pdl_trigger();
    pdl_wait();
    extern __shared__ __align__(16) float sg_smem[];
    float* term = sg_smem;                                  // [max_blocks * GP]
    float* sc = sg_smem + (size_t)a.max_blocks * GP;        // [max_blocks]: scores, then keep flags
    __shared__ float red[4][2 * 32 * GP];
    __shared__ float fin[2][2 * GP];
    __shared__ float nHs[GP];                    // n / H per head (< 0: H = 0, every block scores 1)
    __shared__ int wsum[NW];
    __shared__ int hist[256];
    __shared__ int sel_digit, sel_rem;
    __shared__ float arg_v[NW];
    __shared__ int arg_j[NW];
    __shared__ float nm[NW][GP], nl[NW][GP];     // kept-norm partials per warp and head
    const int seg = blockIdx.x;
    const int b = seg / a.Hkv, kvh = seg - b * a.Hkv;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int h = lane & (GP - 1);
    const int jt = tid / GP;
    const int L = a.ctx_lens[b];
    const bool bad_ctx = L < 0 || L > a.max_blocks * a.P;
    const int nb = bad_ctx ? 0 : (L + a.P - 1) / a.P;
    const long long segbase = (long long)seg * a.max_blocks;
    const float4* st = a.stats + segbase * G;

    // exclusive prefix of one int per thread over the CTA (in thread order);
    // returns it and the total in *tot
    auto scan_excl = [&](int v, int* tot) {
        int x = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x += y;
        }
        if (lane == 31) wsum[wid] = x;
        __syncthreads();
        int before = 0, all = 0;
        for (int u = 0; u < NW; ++u) {
            const int y = wsum[u];
            before += u < wid ? y : 0;
            all += y;
        }
        __syncthreads();
        *tot = all;
        return before + x - v;
    };

    // pass 1: page ids, stale stats, the per-head max
    const int bad = any_bad_page(a.block_table + (long long)b * a.max_blocks, tid, NT, nb, a.num_pages);
    int stale = 0;
    float Mh[1] = {-kInf};
    if (h < G)
        for (int j = jt; j < nb; j += JS) {
            const float x = st[(long long)j * G + h].x;
            stale |= (x != x);                   // NaN max: the scoring pass gave up on this block
            Mh[0] = fmaxf(Mh[0], x);
        }
    const bool bad_page = __syncthreads_or(bad) != 0;
    const bool timed_out = __syncthreads_or(stale) != 0 && !bad_page;
    bool drain = false;
    if (timed_out) {
        // rare: a block marked l - 1 = +inf had a copy in flight when the drain gave up
        int d = 0;
        if (h < G)
            for (int j = jt; j < nb; j += JS) {
                const float4 v = st[(long long)j * G + h];
                d |= (v.x != v.x) && v.y == kInf;
            }
        drain = __syncthreads_or(d) != 0;
    }
    if (a.err && tid == 0) {
        // err was cleared before this kernel; every kv head ORs in its bits
        const uint32_t e = (bad_ctx ? ETI_ERRF_BAD_CTX : 0u) | (bad_page ? ETI_ERRF_BAD_PAGE : 0u) |
                           (timed_out ? ETI_ERRF_TIMEOUT : 0u) | (drain ? ETI_ERRF_DRAIN : 0u);
        if (e) atomicOr(a.err + b, e);
    }
    const int n = (bad_ctx || bad_page || timed_out) ? 0 : nb;
    if (n > 0) {
        head_reduce2<GP, 1, true>(Mh, red[0], fin[0]);
        const float M = Mh[0];
        // pass 2: Z - 1 = sum_b c_b l1_b + sum_{b: m_b < M} c_b + (#blocks at M - 1),
        // c_b = e^{m_b - M} (the blocks at the max are counted, not summed)
        float zs[2] = {0.f, 0.f};
        if (h < G)
            for (int j = jt; j < n; j += JS) {
                const float2 v = *reinterpret_cast<const float2*>(st + (long long)j * G + h);
                const bool top = !(v.x < M);
                const float c = top ? 1.f : exp_le0(v.x - M);
                zs[0] += c * v.y + (top ? 0.f : c);
                zs[1] += top ? 1.f : 0.f;
                term[j * GP + h] = c;
            }
        head_reduce2<GP, 2, false>(zs, red[1], fin[1]);
        const float zm1 = zs[0] + (zs[1] - 1.f);
        const float lZ = log1pf(zm1), iZ = 1.f / (1.f + zm1);
        // pass 3: I_b = e^{m_b - M}[(1 + l1_b)(log Z + M - m_b) - u_b] / Z; H = sum_b I_b
        float Hs[1] = {0.f};
        if (h < G)
            for (int j = jt; j < n; j += JS) {
                const float4 v = st[(long long)j * G + h];
                const float c = term[j * GP + h];
                float t;
                if (a.score_mode == 1) t = c * v.w * iZ;                       // E
                else if (a.score_mode == 2) t = c * (1.f + v.y) * iZ;          // M
                else t = c * ((1.f + v.y) * (lZ + M - v.x) - v.z) * iZ;        // A
                term[j * GP + h] = t;
                Hs[0] += t;
            }
        head_reduce2<GP, 1, false>(Hs, red[2], fin[0]);
        if (tid < GP) nHs[tid] = Hs[0] > 0.f ? (float)n / Hs[0] : -1.f;
        __syncthreads();
    }

    // group scores: thread t takes blocks t, t + NT, ... (a warp reads
    // consecutive blocks' terms with 16-byte loads: few bank conflicts)
    float nh[GP];
#pragma unroll
    for (int hh = 0; hh < GP; ++hh) nh[hh] = hh < G ? nHs[hh] : -kInf;
    float bs = -kInf;                            // this thread's best score and its block
    int bj = 0x7fffffff;
    for (int j = tid; j < n; j += NT) {
        float t[GP];
        if (GP >= 4) {
#pragma unroll
            for (int c = 0; c < GP / 4; ++c) {
                const float4 v = reinterpret_cast<const float4*>(term + j * GP)[c];
                t[4 * c] = v.x; t[4 * c + 1] = v.y; t[4 * c + 2] = v.z; t[4 * c + 3] = v.w;
            }
        } else {
#pragma unroll
            for (int hh = 0; hh < GP; ++hh) t[hh] = term[j * GP + hh];
        }
        float s = -kInf;
#pragma unroll
        for (int hh = 0; hh < G; ++hh) s = fmaxf(s, nh[hh] < 0.f ? 1.f : t[hh] * nh[hh]);
        sc[j] = s;
        if (a.block_score) a.block_score[segbase + j] = s;
        if (s > bs || bj == 0x7fffffff) { bs = s; bj = j; }   // ascending j: the first of equal scores stays
    }
    if (a.block_score)
        for (int j = n + tid; j < a.max_blocks; j += NT) a.block_score[segbase + j] = 0.f;
    __syncthreads();
    // per block from here: thread t takes the run of blocks [j0, j1)
    const int q = (n + NT - 1) / NT;
    const int j0 = min(n, tid * q), j1 = min(n, j0 + q);

    // B_min budget: the first kb blocks by (score desc, index asc)
    const float th = a.theta[b];
    const int kb = min(max(a.B_min, 0), n);
    const bool sel = kb > 1 && kb < n;
    int arg = -1, need = 0;
    uint32_t kth = 0u;
    if (kb == 1 && n > 1) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float ov = __shfl_xor_sync(0xffffffffu, bs, o);
            const int oj = __shfl_xor_sync(0xffffffffu, bj, o);
            if (oj != 0x7fffffff && (bj == 0x7fffffff || ov > bs || (ov == bs && oj < bj))) { bs = ov; bj = oj; }
        }
        if (lane == 0) { arg_v[wid] = bs; arg_j[wid] = bj; }
        __syncthreads();
        for (int u = 0; u < NW; ++u)
            if (arg_j[u] != 0x7fffffff && (bj == 0x7fffffff || arg_v[u] > bs || (arg_v[u] == bs && arg_j[u] < bj))) {
                bs = arg_v[u];
                bj = arg_j[u];
            }
        arg = bj;
    } else if (sel) {
        uint32_t prefix = 0, mask = 0;
        need = kb;
        for (int digit = 3; digit >= 0; --digit) {
            const int shf = digit * 8;
            for (int i = tid; i < 256; i += NT) hist[i] = 0;
            __syncthreads();
            for (int jb = 0; jb < n; jb += NT) {      // the same trip count for every lane
                const int j = jb + tid;
                const uint32_t key = j < n ? order_key(sc[j]) : 0u;
                warp_hist_add(hist, (key >> shf) & 255, j < n && (key & mask) == prefix);
            }
            __syncthreads();
            // bucket where the count from the top reaches `need`
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
            prefix |= (uint32_t)sel_digit << shf;
            mask |= 255u << shf;
            need = sel_rem;
            __syncthreads();
        }
        kth = prefix;
    }
    // keep flags (ties at the k-th key to the lower block index: ranked in
    // thread order, which is block order)
    int neq = 0;
    if (sel)
        for (int j = j0; j < j1; ++j) neq += order_key(sc[j]) == kth;
    int eq_tot;
    int eq_rank = sel ? scan_excl(neq, &eq_tot) : 0;
    int nkeep = 0;
    uint32_t kbits = 0;                          // this run's keep flags (q <= 32 blocks a thread)
    for (int j = j0; j < j1; ++j) {
        const float s = sc[j];
        const uint32_t key = order_key(s);
        bool keep = s >= th || kb >= n || j == arg || (sel && key > kth);
        if (sel && key == kth) keep |= eq_rank++ < need;
        kbits |= keep ? 1u << (j - j0) : 0u;
        nkeep += keep;
    }
    int total;
    int pos = scan_excl(nkeep, &total);          // (its barriers order the score reads above)
    for (int j = j0; j < j1; ++j) {
        const bool keep = (kbits >> (j - j0)) & 1u;
        if (keep) a.kept_idx[segbase + pos++] = j;
        if (a.keep_mask) a.keep_mask[segbase + j] = keep ? 1 : 0;
        sc[j] = keep ? 1.f : 0.f;
    }
    for (int i = total + tid; i < a.max_blocks; i += NT) a.kept_idx[segbase + i] = -1;
    if (a.keep_mask)
        for (int j = n + tid; j < a.max_blocks; j += NT) a.keep_mask[segbase + j] = 0;
    if (tid == 0) a.kept_cnt[seg] = total;

    // softmax normaliser over the kept tokens of each query head: an online
    // (max, sum of (1 + l1) e^{m - max}) over the kept blocks, merged over
    // the lanes of a head and then over the warps in warp order
    if (a.kept_norm) {
        __syncthreads();                         // the keep flags in sc
        float mk = -kInf, lk = 0.f;
        if (h < G)
            for (int j = jt; j < n; j += JS) {
                if (sc[j] == 0.f) continue;
                const float2 v = *reinterpret_cast<const float2*>(st + (long long)j * G + h);
                if (v.x > mk) {
                    lk = (mk == -kInf ? 0.f : lk * exp_le0(mk - v.x)) + (1.f + v.y);
                    mk = v.x;
                } else {
                    lk += (1.f + v.y) * exp_le0(v.x - mk);
                }
            }
        auto merge = [](float& m1, float& l1, float m2, float l2) {
            if (m2 == -kInf) return;
            if (m1 == -kInf) { m1 = m2; l1 = l2; return; }
            const float mm = fmaxf(m1, m2);
            l1 = l1 * exp_le0(m1 - mm) + l2 * exp_le0(m2 - mm);
            m1 = mm;
        };
#pragma unroll
        for (int o = 16; o >= GP; o >>= 1) {
            const float om = __shfl_xor_sync(0xffffffffu, mk, o);
            const float ol = __shfl_xor_sync(0xffffffffu, lk, o);
            merge(mk, lk, om, ol);               // (the two sides agree: the sum commutes)
        }
        if (lane < GP) { nm[wid][lane] = mk; nl[wid][lane] = lk; }
        __syncthreads();
        if (tid < G) {
            float m1 = -kInf, l1 = 0.f;
            for (int u = 0; u < NW; ++u) merge(m1, l1, nm[u][tid], nl[u][tid]);
            float* kn = a.kept_norm + ((long long)b * a.Hq + kvh * a.g + tid) * 2;
            kn[0] = m1;
            kn[1] = l1;
        }
    }
}

// Launch of the segment kernel (programmatic dependent launch): 128, 256 or
// 512 threads, about 16 block-heads of the longest segment a thread.
template <int G, int NT>
cudaError_t launch_seg_nt(int segs, cudaStream_t stream, const FinArgs& a) {
    constexpr int GP = FlatGP<G>::v;
    auto k = prune_finalize_seg_kernel<G, NT>;
    const size_t smem = (size_t)a.max_blocks * (GP + 1) * 4;
    if (smem > 48 * 1024) cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    return eti_launch_pdl(k, dim3(segs), dim3(NT), smem, stream, a);
}
template <int G>
cudaError_t launch_seg(int segs, cudaStream_t stream, const FinArgs& a) {
    constexpr int GP = FlatGP<G>::v;
    const long long slots = (long long)a.max_blocks * GP;
    if (slots <= 128 * 16) return launch_seg_nt<G, 128>(segs, stream, a);
    if (slots <= 256 * 16) return launch_seg_nt<G, 256>(segs, stream, a);
    return launch_seg_nt<G, 512>(segs, stream, a);
}

// Launch of the wide kernel for `segs` segments, kCl CTAs of NT threads per
// segment (a cluster), with programmatic dependent launch.
template <int G, int NT, bool kTerm, int kCl>
cudaError_t launch_wide(int segs, size_t smem, cudaStream_t stream, const FinArgs& a) {
    auto k = prune_finalize_wide_kernel<G, NT, kTerm, kCl>;
    if (smem > 48 * 1024) cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(segs * kCl);
    cfg.blockDim = dim3(NT);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = kCl;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = kCl > 1 ? 2 : 1;
    return cudaLaunchKernelEx(&cfg, k, a);
}

// The launch shape: long segments fewer than half the SMs take a pair of
// 1024-thread CTAs each (more threads per segment); the rest one 512-thread
// CTA each, two CTAs per SM where the shared memory allows (on 1024 segments
// of up to 2048 blocks x 8 heads: 157 us against 201 us with one 1024-thread
// CTA per SM; 256-thread CTAs took 313 us).  The term cache is used where it
// fits, the share cache only where it leaves room for two CTAs per SM.
template <int G>
cudaError_t launch_wide_shape(const FinArgs& a, int segs, int sms, cudaStream_t stream) {
    constexpr int GP = FlatGP<G>::v;
    const size_t smem_t = (size_t)a.max_blocks * 4 * (1 + GP), smem_s = (size_t)a.max_blocks * 4;
    const size_t smem_ts = smem_t + (size_t)a.max_blocks * 4 * GP;
    const bool term = !a.given && smem_t <= kWideSmemMax;
    FinArgs b = a;
    if (2 * segs <= sms && a.max_blocks > (kWideThreads / GP) * kFlatPer) {
        b.share_cache = term && smem_ts <= kWideSmemMax;
        const size_t smem = term ? (b.share_cache ? smem_ts : smem_t) : smem_s;
        const cudaError_t e = term ? launch_wide<G, kWideThreads, true, 2>(segs, smem, stream, b)
                                   : launch_wide<G, kWideThreads, false, 2>(segs, smem, stream, b);
        if (e == cudaSuccess) return e;
        (void)cudaGetLastError();   // cluster launch refused: one CTA per segment
    }
    // the rule mode with the terms of a segment in shared memory (and at most
    // 32 blocks per thread in the per-block passes): the segment kernel
    if (!a.given && a.theta && (size_t)a.max_blocks * (GP + 1) * 4 <= kWideSmemMax / 2 &&
        a.max_blocks <= 512 * 32)
        return launch_seg<G>(segs, stream, a);
    b.share_cache = term && smem_ts <= kWideSmemMax / 2;
    const size_t smem = term ? (b.share_cache ? smem_ts : smem_t) : smem_s;
    return term ? launch_wide<G, kWideThreads / 2, true, 1>(segs, smem, stream, b)
                : launch_wide<G, kWideThreads / 2, false, 1>(segs, smem, stream, b);
}

}  // namespace eti

// Host entry of the wide keep-set kernel (the caller has cleared a.err).
cudaError_t eti_launch_prune_wide(const eti::FinArgs& a, int segs, int sms, cudaStream_t stream) {
    using namespace eti;
    switch (a.g) {
        case 1: return launch_wide_shape<1>(a, segs, sms, stream);
        case 2: return launch_wide_shape<2>(a, segs, sms, stream);
        case 3: return launch_wide_shape<3>(a, segs, sms, stream);
        case 4: return launch_wide_shape<4>(a, segs, sms, stream);
        case 5: return launch_wide_shape<5>(a, segs, sms, stream);
        case 6: return launch_wide_shape<6>(a, segs, sms, stream);
        case 7: return launch_wide_shape<7>(a, segs, sms, stream);
        case 8: return launch_wide_shape<8>(a, segs, sms, stream);
        default: return cudaErrorInvalidValue;
    }
}
