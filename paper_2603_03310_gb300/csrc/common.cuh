// common.cuh -- device helpers shared by the libeti kernels (sm_103a).
//
// Thin wrappers around single PTX instructions: streaming 128-bit loads, the
// MUFU exp2 / log2 approximations, the legacy bf16 tensor-core tile
// (mma.sync m16n8k16) and warp shuffles.  No math routine is re-derived here:
// ex2/lg2 are the hardware approximations, used where the callers' error
// analysis allows them, and the accurate libdevice functions are called where
// it does not.
#pragma once

#include <cstdint>
#include <type_traits>

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "../../include/eti.h"

namespace eti {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr float kInf = __builtin_huge_valf();

// 16-byte read-only load that does not allocate in L1 (data read once).
__device__ __forceinline__ uint4 ldg_stream_u4(const void* p) {
    uint4 r;
    asm("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
        : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
        : "l"(p));
    return r;
}

__device__ __forceinline__ float4 ldg_stream_f4(const float* p) {
    float4 r;
    asm("ld.global.nc.L1::no_allocate.v4.f32 {%0,%1,%2,%3}, [%4];"
        : "=f"(r.x), "=f"(r.y), "=f"(r.z), "=f"(r.w)
        : "l"(p));
    return r;
}

__device__ __forceinline__ uint2 ldg_stream_u2(const void* p) {
    uint2 r;
    asm("ld.global.nc.L1::no_allocate.v2.u32 {%0,%1}, [%2];"
        : "=r"(r.x), "=r"(r.y)
        : "l"(p));
    return r;
}

// 2^x, hardware approximation (MUFU.EX2), denormal results flushed to zero.
__device__ __forceinline__ float fast_ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Whether any page id row[j], j = first, first + stride, ... < n, lies
// outside [0, num_pages).  Eight loads per thread are issued before any is
// tested, so a long row costs a few memory round trips, not one per id.
__device__ __forceinline__ bool any_bad_page(const int32_t* row, int first, int stride, int n,
                                             long long num_pages) {
    constexpr int kU = 8;
    bool bad = false;
    for (int j0 = first; j0 < n; j0 += kU * stride) {
        int pg[kU];
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            const int j = j0 + u * stride;
            pg[u] = j < n ? __ldg(row + j) : 0;
        }
#pragma unroll
        for (int u = 0; u < kU; ++u)
            bad |= j0 + u * stride < n && (pg[u] < 0 || (long long)pg[u] >= num_pages);
    }
    return bad;
}

// 1/x, hardware approximation (MUFU.RCP); 1/0 = +inf.
__device__ __forceinline__ float fast_rcp(float x) {
    float y;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// log2(x), hardware approximation (MUFU.LG2).
__device__ __forceinline__ float fast_lg2(float x) {
    float y;
    asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// D += A * B on one m16n8k16 bf16 tile with fp32 accumulators.
// Fragment ownership (lane = 4 * grp + t):
//   A (16x16, row-major): a0 = A[grp][2t..2t+1], a1 = A[grp+8][2t..2t+1],
//                         a2 = A[grp][2t+8..2t+9], a3 = A[grp+8][2t+8..2t+9]
//   B (16x8, col-major):  b0 = B[2t..2t+1][grp], b1 = B[2t+8..2t+9][grp]
//   D (16x8):             d0,d1 = D[grp][2t..2t+1], d2,d3 = D[grp+8][2t..2t+1]
__device__ __forceinline__ void mma_bf16_16x8x16(float (&d)[4], uint32_t a0, uint32_t a1,
                                                 uint32_t a2, uint32_t a3, uint32_t b0,
                                                 uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
        "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Pack two fp32 values into a bf16x2 register (round to nearest even);
// `lo` lands in the low half.
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

// Low / high bf16 halves of two registers combined into one register.
__device__ __forceinline__ uint32_t lo_halves(uint32_t a, uint32_t b) { return __byte_perm(a, b, 0x5410); }
__device__ __forceinline__ uint32_t hi_halves(uint32_t a, uint32_t b) { return __byte_perm(a, b, 0x7632); }

// Bulk prefetch of `bytes` (a multiple of 16, 16-byte aligned source) into L2;
// no destination, no completion to wait for.
__device__ __forceinline__ void prefetch_l2_bulk(const void* p, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" :: "l"(p), "r"(bytes) : "memory");
}

// ---- mbarrier + TMA (cp.async.bulk.tensor) ----------------------------------

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" :: "r"(bar), "r"(count) : "memory");
}
// make barrier initialisation visible to the async (TMA) proxy
__device__ __forceinline__ void fence_mbar_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
// order this thread's earlier generic shared-memory accesses before later
// async-proxy (TMA) writes to the same buffer
__device__ __forceinline__ void fence_proxy_async() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" :: "r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" :: "r"(bar) : "memory");
}
// Bounded wait for the phase of parity `parity` to complete: returns false
// after `max_iters` unsuccessful polls (each poll may suspend the thread for
// a short, hardware-defined time), so a wait can never hang the GPU.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, int max_iters) {
    for (int it = 0; it < max_iters; ++it) {
        uint32_t done;
        asm volatile(
            "{\n\t.reg .pred p;\n\t"
            "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
            "selp.u32 %0, 1, 0, p;\n\t}"
            : "=r"(done) : "r"(bar), "r"(parity) : "memory");
        if (done) return true;
    }
    return false;
}
// 2-D tiled TMA load of one box into shared memory, completing on `bar`.
// x (the inner coordinate) must be a multiple of 16 bytes / element size.
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const void* tmap, int x, int y, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];"
        :: "r"(dst), "l"(tmap), "r"(x), "r"(y), "r"(bar) : "memory");
}
// 1-D bulk copy global -> shared (16-byte aligned addresses, size multiple of 16)
__device__ __forceinline__ void bulk_load_1d(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
        :: "r"(dst), "l"(src), "r"(bytes), "r"(bar) : "memory");
}

// Four 8x8 b16 matrices from shared memory, each transposed (ldmatrix .trans):
// lane l gives the address of row l % 8 of matrix l / 8 (16 contiguous bytes);
// register i of lane (4 g + t) then holds rows 2t, 2t+1 of column g of matrix i.
__device__ __forceinline__ void ldsm_x4_trans(uint32_t (&r)[4], uint32_t addr) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]) : "r"(addr) : "memory");
}
__device__ __forceinline__ void sts_zero_u4(uint32_t addr) {
    asm volatile("st.shared.v4.u32 [%0], {%1, %1, %1, %1};" :: "r"(addr), "r"(0u) : "memory");
}

// Offset of the 16-byte chunk `chunk` of row `row` inside a TMA box with
// 128-byte rows and the 128-byte swizzle (chunk index xor row mod 8).
__device__ __forceinline__ uint32_t swz128(int row, int chunk) {
    return (uint32_t)(row * 128 + ((chunk ^ (row & 7)) << 4));
}

// Shared-state-space address of a shared-memory pointer.
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// Asynchronous global -> shared copies (cp.async): `bytes` are copied when
// `valid`, otherwise the destination is zero-filled and nothing is read.
__device__ __forceinline__ void cp_async_16(uint32_t dst, const void* src, bool valid) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;"
                 :: "r"(dst), "l"(src), "r"(valid ? 16 : 0) : "memory");
}
__device__ __forceinline__ void cp_async_8(uint32_t dst, const void* src, bool valid) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8, %2;"
                 :: "r"(dst), "l"(src), "r"(valid ? 8 : 0) : "memory");
}
__device__ __forceinline__ void cp_async_4(uint32_t dst, const void* src, bool valid) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;"
                 :: "r"(dst), "l"(src), "r"(valid ? 4 : 0) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
// wait until at most N of this thread's committed groups are still in flight
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" :: "n"(N) : "memory"); }

__device__ __forceinline__ uint4 lds_u4(uint32_t a) {
    uint4 r;
    asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w) : "r"(a));
    return r;
}
__device__ __forceinline__ uint2 lds_u2(uint32_t a) {
    uint2 r;
    asm volatile("ld.shared.v2.u32 {%0,%1}, [%2];" : "=r"(r.x), "=r"(r.y) : "r"(a));
    return r;
}
__device__ __forceinline__ float lds_f32(uint32_t a) {
    float r;
    asm volatile("ld.shared.f32 %0, [%1];" : "=f"(r) : "r"(a));
    return r;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ int warp_sum_i(int v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// ---- thread-block clusters (distributed shared memory) ----------------------

__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
// Barrier over every thread of every CTA of the cluster (release / acquire:
// shared-memory writes before it are visible to the cluster after it).
__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\t"
                 "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// Loads from the same shared-memory variable of CTA `rank` of the cluster.
__device__ __forceinline__ float ld_cluster_f32(const void* p, uint32_t rank) {
    uint32_t a;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(a) : "r"(smem_u32(p)), "r"(rank));
    float v;
    asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(a) : "memory");
    return v;
}
__device__ __forceinline__ int ld_cluster_s32(const void* p, uint32_t rank) {
    uint32_t a;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(a) : "r"(smem_u32(p)), "r"(rank));
    int v;
    asm volatile("ld.shared::cluster.s32 %0, [%1];" : "=r"(v) : "r"(a) : "memory");
    return v;
}

// hist[bin] += 1 for every lane with `on`, one shared-memory atomic per
// distinct bin of the warp (every lane of the warp must call it together)
__device__ __forceinline__ void warp_hist_add(int* hist, uint32_t bin, bool on) {
    const uint32_t act = __ballot_sync(0xffffffffu, on);
    if (on) {
        const uint32_t peers = __match_any_sync(act, bin);
        if ((threadIdx.x & 31) == (uint32_t)(__ffs(peers) - 1)) atomicAdd(hist + bin, __popc(peers));
    }
}

__host__ __device__ __forceinline__ int ceil_div(int a, int b) { return (a + b - 1) / b; }

// Blocks of a sequence with context length L (0 for an invalid length, which
// the finalizing kernels report).
__device__ __forceinline__ int seq_blocks(int L, int P, int max_blocks) {
    if (L <= 0 || L > max_blocks * P) return 0;
    return (L + P - 1) / P;
}

// Default number of polls before a wait for a tile copy gives up; the
// kernels take their limit as an argument (eti_set_wait_limit), and the
// drain after a timeout always uses this default.
constexpr int kMaxWaitIters = 1 << 20;

// Programmatic dependent launch: let the next kernel in the stream be
// scheduled now (it still waits for this grid to finish before reading our
// results), and wait for the previous grid's results before reading them.
// Both are no-ops when the kernel was launched without the attribute.
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

}  // namespace eti

// Launch with programmatic stream serialization (overlaps this kernel's
// launch with the previous kernel's tail).
template <typename... KArgs, typename... Args>
inline cudaError_t eti_launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                                  cudaStream_t stream, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// Host: the current wait limit for the tile waits (eti_set_wait_limit).
int eti_wait_limit();

// Host: a 2-D bf16 tensor map over a [rows][D] array with boxes of
// 16 rows x 64 elements (128 bytes) and the 128-byte swizzle.
int eti_make_kv_tensor_map(CUtensorMap* map, const void* base, long long rows, int D);
