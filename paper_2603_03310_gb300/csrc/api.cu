// api.cu -- the extern "C" boundary of libeti: argument validation, workspace
// layout and the launch sequence of each entry point.  Declarations and the
// full contract are in include/eti.h.
#include <atomic>
#include <cstring>

#include "common.cuh"

// launchers (defined next to their kernels)
int eti_launch_entropy_temp_sample(const float* logits, int B, int V, long long ld,
                                   const float* T_in, const float* H_prev, float* tau,
                                   const float* H_target, const eti_ctrl_params* p,
                                   uint64_t seed, uint64_t offset, uint64_t* offset_dev,
                                   int32_t* tok, float* H, float* T_out, float* dH,
                                   float* theta_next, float* surprisal,
                                   const eti_surp_store* store, uint32_t* err, void* scratch,
                                   cudaStream_t stream);
size_t eti_entropy_partial_bytes(int B);
int eti_launch_schedule(const float* dH, float* ema, const int32_t* kept_cnt, int Hkv, int P,
                        const int32_t* ctx_lens, const float* urgency, const eti_sched_params* p,
                        int B, int budget, float* priority, uint8_t* admit, cudaStream_t stream);
int eti_launch_topk_entropy(const float* logits, int B, int V, long long ld, const float* T_in,
                            int k, float* H_tilde, float* H_hat, float* tail_mass, uint32_t* err,
                            cudaStream_t stream);
int eti_launch_score_blocks(const uint16_t* q, const uint16_t* k_cache, const int32_t* block_table,
                            const int32_t* ctx_lens, int B, int Hq, int Hkv, int D, int P,
                            int max_blocks, long long num_pages, float scale, const float* tok_surp,
                            float* token_scores, float4* stats, cudaStream_t stream);
int eti_launch_prune_finalize(const float4* stats, const int32_t* ctx_lens, const int32_t* block_table,
                              long long num_pages, int B, int Hq, int Hkv, int P, int max_blocks,
                              const float* theta, int B_min, int score_mode, int given,
                              const uint8_t* given_mask,
                              const int32_t* given_idx, const int32_t* given_cnt, uint8_t* keep_mask,
                              int32_t* kept_idx, int32_t* kept_cnt, float* block_score,
                              float* kept_norm, uint32_t* err, cudaStream_t stream);
int eti_launch_decode(const uint16_t* v_cache, const int32_t* block_table, const int32_t* ctx_lens,
                      const int32_t* kept_idx, const int32_t* kept_cnt, const float* token_scores,
                      const float* kept_norm, int B, int Hq, int Hkv, int D, int P, int max_blocks,
                      long long num_pages, uint16_t* out, uint32_t* err, int* plan_cum,
                      int* plan_info, int* plan_warp_seg, int* plan_ticket, float* partial,
                      int nwarps, cudaStream_t stream);
int eti_decode_nwarps(int D, int g);

// cuTensorMapEncodeTiled, fetched from the driver at first use (no link
// dependency on libcuda).
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

int eti_make_kv_tensor_map(CUtensorMap* map, const void* base, long long rows, int D) {
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess || !p)
            return ETI_ERR_CUDA;
        fn = reinterpret_cast<EncodeTiledFn>(p);
    }
    if (rows <= 0 || (rows >> 32) != 0) return ETI_ERR_SHAPE;
    const cuuint64_t dims[2] = {(cuuint64_t)D, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)D * 2};
    const cuuint32_t box[2] = {64, 16};
    const cuuint32_t estr[2] = {1, 1};
    const CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims,
                          strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                          CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? ETI_OK : ETI_ERR_CUDA;
}

namespace {

// polls before a tile wait gives up (eti_set_wait_limit)
std::atomic<int> g_wait_limit{eti::kMaxWaitIters};

constexpr int kMaxB = 8192;
constexpr int kMaxBlocks = 32768;
constexpr long long kMaxUnits = 1LL << 30;   // B * Hkv * max_blocks

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }
size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

int check_attn_shape(int B, int Hq, int Hkv, int D, int P, int max_blocks, long long num_pages) {
    if (B < 0 || B > kMaxB || Hq <= 0 || Hkv <= 0 || max_blocks <= 0 || num_pages < 0)
        return ETI_ERR_SHAPE;
    if (Hq % Hkv != 0) return ETI_ERR_SHAPE;
    if (Hq / Hkv > 8 || max_blocks > kMaxBlocks) return ETI_ERR_UNSUPPORTED;
    if (!((D == 64 || D == 128) && (P == 16 || P == 32))) return ETI_ERR_UNSUPPORTED;
    if ((long long)max_blocks * P > 0x7fffffffLL) return ETI_ERR_SHAPE;
    // the kernels count (sequence, kv head, block) units and their prefix
    // sums in 32-bit ints, and a TMA row coordinate (page * Hkv + head) * P
    // is a signed 32-bit value
    if ((long long)B * Hkv * max_blocks > kMaxUnits) return ETI_ERR_UNSUPPORTED;
    if (num_pages > 0x7fffffffLL / ((long long)Hkv * P)) return ETI_ERR_UNSUPPORTED;
    return ETI_OK;
}

// Carves consecutive 256-byte aligned regions out of a workspace.
struct Carver {
    char* base;
    size_t off = 0;
    explicit Carver(void* p) : base(static_cast<char*>(p)) {}
    template <class T>
    T* take(size_t count) {
        T* p = reinterpret_cast<T*>(base ? base + off : nullptr);
        off = align256(off + count * sizeof(T));
        return p;
    }
};

struct DecodeWs {
    float* scores; float4* stats; int32_t* kidx; int32_t* kcnt; float* knorm;
    int* cum; int* info; int* warp_seg; int* ticket; float* partial;
};

DecodeWs carve_decode(void* ws, int B, int Hq, int Hkv, int D, int P, int max_blocks,
                      int have_scores, int nwarps, size_t* bytes) {
    Carver c(ws);
    DecodeWs w{};
    const size_t g = Hq / Hkv, nseg = (size_t)B * Hkv;
    if (!have_scores) {
        w.scores = c.take<float>(nseg * max_blocks * P * g);
        w.stats = c.take<float4>(nseg * max_blocks * g);
        w.kidx = c.take<int32_t>(nseg * max_blocks);
        w.kcnt = c.take<int32_t>(nseg);
        w.knorm = c.take<float>((size_t)B * Hq * 2);
    }
    w.cum = c.take<int>(nseg + 1);
    w.info = c.take<int>(4);   // total kept blocks, share per warp
    w.warp_seg = c.take<int>(nwarps);
    w.ticket = c.take<int>(nseg);
    w.partial = c.take<float>(((size_t)nwarps + nseg) * g * D);
    *bytes = c.off;
    return w;
}

}  // namespace

extern "C" {

void eti_ctrl_defaults(eti_ctrl_params* p) {
    if (!p) return;
    p->eta = 0.1f;
    p->sign = -1.0f;
    p->T_min = 0.05f;
    p->T_max = 5.0f;
    p->eps_H = 0.0f;
    p->H_min = 0.0f;
    p->theta_user = __builtin_huge_valf();
    p->theta_hi = 1.0f;
    p->T_cal = 1.0f;
    p->rho_T = 0.0f;
    p->dtheta = 0.0f;
}

const char* eti_version(void) { return "libeti 0.2.0 (sm_103a)"; }

int64_t eti_set_wait_limit(int64_t polls) {
    const int v = polls < 0 ? eti::kMaxWaitIters : (int)std::min<int64_t>(polls, 0x7fffffff);
    return g_wait_limit.exchange(v);
}

const char* eti_status_string(int s) {
    switch (s) {
        case ETI_OK: return "ok";
        case ETI_ERR_NULL: return "a required pointer is NULL";
        case ETI_ERR_SHAPE: return "a size is out of range or inconsistent";
        case ETI_ERR_UNSUPPORTED: return "shape not supported by this library";
        case ETI_ERR_WORKSPACE: return "workspace missing or too small";
        case ETI_ERR_CUDA: return "CUDA launch failed";
        case ETI_ERR_TIMEOUT: return "a device-side wait gave up (reserved: reported per sequence in err_flags)";
        case ETI_ERR_TOO_LARGE: return "problem exceeds the fixed scratch of the no-allocation entry point";
        case ETI_ERR_ALIGN: return "a bf16 tensor is not 16-byte aligned";
        default: return "unknown status";
    }
}

size_t eti_entropy_temp_sample_workspace_size(int B, int V) {
    if (B < 0 || B > 65535 || V < 1) return 0;
    return align256(eti_entropy_partial_bytes(B));
}

int eti_entropy_temp_sample(const float* logits, int B, int V, int64_t ld,
                            const float* T_in, const float* H_prev, float* tau,
                            const float* H_target, const eti_ctrl_params* params,
                            uint64_t seed, uint64_t offset, uint64_t* offset_dev,
                            int32_t* tok, float* H, float* T_out,
                            float* dH, float* theta_next, float* tok_surprisal,
                            const eti_surp_store* surp_store,
                            uint32_t* err_flags, void* ws, size_t ws_bytes, void* stream) {
    if (B < 0 || B > 65535 || V < 1 || ld < V) return ETI_ERR_SHAPE;
    if (B == 0) return ETI_OK;
    if (!logits || !T_in || !H_prev || !tau || !H_target || !params || !tok || !H || !T_out ||
        !err_flags)
        return ETI_ERR_NULL;
    if (surp_store && (!surp_store->store || !surp_store->slot_mapping)) return ETI_ERR_NULL;
    if (!ws || ws_bytes < eti_entropy_temp_sample_workspace_size(B, V)) return ETI_ERR_WORKSPACE;
    if ((reinterpret_cast<uintptr_t>(ws) & 3) != 0) return ETI_ERR_WORKSPACE;
    return eti_launch_entropy_temp_sample(logits, B, V, (long long)ld, T_in, H_prev, tau, H_target,
                                          params, seed, offset, offset_dev, tok, H, T_out, dH,
                                          theta_next, tok_surprisal, surp_store, err_flags, ws,
                                          (cudaStream_t)stream);
}

int eti_topk_entropy(const float* logits, int B, int V, int64_t ld, const float* T_in, int k,
                     float* H_tilde, float* H_hat, float* tail_mass, uint32_t* err_flags,
                     void* stream) {
    if (B < 0 || B > 65535 || V < 1 || ld < V || k < 1) return ETI_ERR_SHAPE;
    if (B == 0) return ETI_OK;
    if (!logits || !T_in || !H_tilde || !H_hat || !err_flags) return ETI_ERR_NULL;
    return eti_launch_topk_entropy(logits, B, V, (long long)ld, T_in, k, H_tilde, H_hat, tail_mass,
                                   err_flags, (cudaStream_t)stream);
}

void eti_sched_defaults(eti_sched_params* p) {
    if (!p) return;
    p->lambda = 0.9f;
    p->alpha = 1e-3f;
    p->beta = 1e-3f;
    p->gamma = 1.0f;
    p->den_min = 1e-6f;
}

int eti_schedule(const float* dH, float* ema, const int32_t* kept_cnt, int Hkv, int P,
                 const int32_t* ctx_lens, const float* urgency, const eti_sched_params* params,
                 int B, int budget, float* priority, uint8_t* admit_mask, void* stream) {
    if (B < 0 || B > 65535 || (kept_cnt && (Hkv < 1 || P < 1))) return ETI_ERR_SHAPE;
    if (B == 0) return ETI_OK;
    if (!dH || !ema || !params || !priority || !admit_mask) return ETI_ERR_NULL;
    return eti_launch_schedule(dH, ema, kept_cnt, Hkv, P, ctx_lens, urgency, params, B, budget,
                               priority, admit_mask, (cudaStream_t)stream);
}

size_t eti_score_prune_workspace_size(int B, int Hq, int Hkv, int D, int P, int max_blocks) {
    if (check_attn_shape(B, Hq, Hkv, D, P, max_blocks, 0) != ETI_OK) return 0;
    Carver c(nullptr);
    c.take<float4>((size_t)B * Hq * max_blocks);
    return c.off;
}

int eti_score_prune_blocks(const eti_bf16* q, const eti_bf16* k_cache,
                           const int32_t* block_table, const int32_t* ctx_lens,
                           int B, int Hq, int Hkv, int D, int P, int max_blocks,
                           int64_t num_pages, float scale,
                           const float* theta, int B_min, int score_mode, const float* tok_surp,
                           uint8_t* keep_mask, int32_t* kept_idx, int32_t* kept_cnt,
                           float* block_score, float* token_scores, float* kept_norm,
                           uint32_t* err_flags, void* ws, size_t ws_bytes, void* stream) {
    int st = check_attn_shape(B, Hq, Hkv, D, P, max_blocks, num_pages);
    if (st != ETI_OK) return st;
    if (score_mode < ETI_SCORE_A || score_mode > ETI_SCORE_M) return ETI_ERR_UNSUPPORTED;
    if (B == 0) return ETI_OK;
    if (score_mode == ETI_SCORE_E && !tok_surp) return ETI_ERR_NULL;
    if (!q || !k_cache || !block_table || !ctx_lens || !theta || !keep_mask || !kept_idx ||
        !kept_cnt || !err_flags)
        return ETI_ERR_NULL;
    if ((token_scores == nullptr) != (kept_norm == nullptr)) return ETI_ERR_NULL;
    if (!aligned16(q) || !aligned16(k_cache)) return ETI_ERR_ALIGN;
    const size_t need = eti_score_prune_workspace_size(B, Hq, Hkv, D, P, max_blocks);
    if (!ws || ws_bytes < need) return ETI_ERR_WORKSPACE;
    cudaStream_t s = (cudaStream_t)stream;
    float4* stats = static_cast<float4*>(ws);
    st = eti_launch_score_blocks(q, k_cache, block_table, ctx_lens, B, Hq, Hkv, D, P, max_blocks,
                                 (long long)num_pages, scale,
                                 score_mode == ETI_SCORE_E ? tok_surp : nullptr, token_scores, stats, s);
    if (st != ETI_OK) return st;
    return eti_launch_prune_finalize(stats, ctx_lens, block_table, (long long)num_pages, B, Hq, Hkv,
                                     P, max_blocks, theta, B_min, score_mode, 0, nullptr, nullptr, nullptr,
                                     keep_mask, kept_idx, kept_cnt, block_score, kept_norm,
                                     err_flags, s);
}

int eti_score_blocks(const eti_bf16* q, const eti_bf16* k_cache, const int32_t* block_table,
                     const int32_t* ctx_lens, int B, int Hq, int Hkv, int D, int P,
                     int max_blocks, int64_t num_pages, float scale, const float* tok_surp,
                     float* token_scores, float* block_stats, void* stream) {
    int st = check_attn_shape(B, Hq, Hkv, D, P, max_blocks, num_pages);
    if (st != ETI_OK) return st;
    if (B == 0) return ETI_OK;
    if (!q || !k_cache || !block_table || !ctx_lens || !block_stats) return ETI_ERR_NULL;
    if (!aligned16(q) || !aligned16(k_cache) || !aligned16(block_stats)) return ETI_ERR_ALIGN;
    return eti_launch_score_blocks(q, k_cache, block_table, ctx_lens, B, Hq, Hkv, D, P, max_blocks,
                                   (long long)num_pages, scale, tok_surp, token_scores,
                                   reinterpret_cast<float4*>(block_stats), (cudaStream_t)stream);
}

int eti_prune_blocks(const float* block_stats, const int32_t* block_table, const int32_t* ctx_lens,
                     int B, int Hq, int Hkv, int D, int P, int max_blocks, int64_t num_pages,
                     const float* theta, int B_min, int score_mode, uint8_t* keep_mask,
                     int32_t* kept_idx, int32_t* kept_cnt, float* block_score, float* kept_norm,
                     uint32_t* err_flags, void* stream) {
    int st = check_attn_shape(B, Hq, Hkv, D, P, max_blocks, num_pages);
    if (st != ETI_OK) return st;
    if (score_mode < ETI_SCORE_A || score_mode > ETI_SCORE_M) return ETI_ERR_UNSUPPORTED;
    if (B == 0) return ETI_OK;
    if (!block_stats || !block_table || !ctx_lens || !theta || !keep_mask || !kept_idx ||
        !kept_cnt || !err_flags)
        return ETI_ERR_NULL;
    if (!aligned16(block_stats)) return ETI_ERR_ALIGN;
    return eti_launch_prune_finalize(reinterpret_cast<const float4*>(block_stats), ctx_lens,
                                     block_table, (long long)num_pages, B, Hq, Hkv, P, max_blocks,
                                     theta, B_min, score_mode, 0, nullptr, nullptr, nullptr, keep_mask, kept_idx,
                                     kept_cnt, block_score, kept_norm, err_flags,
                                     (cudaStream_t)stream);
}

size_t eti_paged_decode_workspace_size(int B, int Hq, int Hkv, int D, int P, int max_blocks,
                                       int have_scores) {
    if (check_attn_shape(B, Hq, Hkv, D, P, max_blocks, 0) != ETI_OK) return 0;
    size_t bytes = 0;
    carve_decode(nullptr, B, Hq, Hkv, D, P, max_blocks, have_scores, eti_decode_nwarps(D, Hq / Hkv), &bytes);
    return bytes;
}

int eti_paged_decode(const eti_bf16* q, const eti_bf16* k_cache, const eti_bf16* v_cache,
                     const int32_t* block_table, const int32_t* ctx_lens,
                     int B, int Hq, int Hkv, int D, int P, int max_blocks,
                     int64_t num_pages, float scale,
                     const uint8_t* keep_mask, const int32_t* kept_idx, const int32_t* kept_cnt,
                     const float* token_scores, const float* kept_norm,
                     eti_bf16* out, uint32_t* err_flags,
                     void* ws, size_t ws_bytes, void* stream) {
    int st = check_attn_shape(B, Hq, Hkv, D, P, max_blocks, num_pages);
    if (st != ETI_OK) return st;
    if (B == 0) return ETI_OK;
    const bool have_lists = kept_idx && kept_cnt;
    const bool have_scores = token_scores && kept_norm && have_lists;
    if (!v_cache || !block_table || !ctx_lens || !out || !err_flags) return ETI_ERR_NULL;
    if (!have_scores && (!q || !k_cache)) return ETI_ERR_NULL;
    if (!aligned16(v_cache) || !aligned16(out) || (have_scores && !aligned16(token_scores)) ||
        (!have_scores && (!aligned16(q) || !aligned16(k_cache))))
        return ETI_ERR_ALIGN;
    const int nwarps = eti_decode_nwarps(D, Hq / Hkv);
    size_t need = 0;
    carve_decode(nullptr, B, Hq, Hkv, D, P, max_blocks, have_scores, nwarps, &need);
    if (!ws || ws_bytes < need) return ETI_ERR_WORKSPACE;
    DecodeWs w = carve_decode(ws, B, Hq, Hkv, D, P, max_blocks, have_scores, nwarps, &need);
    cudaStream_t s = (cudaStream_t)stream;
    if (!have_scores) {
        st = eti_launch_score_blocks(q, k_cache, block_table, ctx_lens, B, Hq, Hkv, D, P,
                                     max_blocks, (long long)num_pages, scale, nullptr, w.scores,
                                     w.stats, s);
        if (st != ETI_OK) return st;
        st = eti_launch_prune_finalize(w.stats, ctx_lens, block_table, (long long)num_pages, B, Hq,
                                       Hkv, P, max_blocks, nullptr, 0, ETI_SCORE_A, 1, keep_mask,
                                       have_lists ? kept_idx : nullptr,
                                       have_lists ? kept_cnt : nullptr, nullptr, w.kidx, w.kcnt,
                                       nullptr, w.knorm, nullptr, s);
        if (st != ETI_OK) return st;
        token_scores = w.scores;
        kept_norm = w.knorm;
        kept_idx = w.kidx;
        kept_cnt = w.kcnt;
    }
    return eti_launch_decode(v_cache, block_table, ctx_lens, kept_idx, kept_cnt, token_scores,
                             kept_norm, B, Hq, Hkv, D, P, max_blocks, (long long)num_pages, out,
                             err_flags, w.cum, w.info, w.warp_seg, w.ticket, w.partial, nwarps, s);
}

}  // extern "C"

int eti_wait_limit() { return g_wait_limit.load(std::memory_order_relaxed); }
