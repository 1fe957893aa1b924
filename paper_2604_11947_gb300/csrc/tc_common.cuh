// tc_common.cuh -- sm_103a building blocks: mbarriers with bounded waits, TMA (tiled bulk
// tensor copies), tcgen05 MMA / TMEM, and the shared-memory matrix descriptors.
//
// Every wait in this file gives up after kWaitNs nanoseconds of wall time, records an error
// code in g_resbm_device_error and returns false, so a logic error cannot leave a kernel
// spinning forever.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace resbm {
namespace tc {

// Error word written by the kernels of the one translation unit that includes this header
// (0 = no error); the host reads it with cudaMemcpyFromSymbol from that unit.
static __device__ unsigned int g_resbm_device_error = 0;

enum : unsigned {
    kErrWaitTimeout = 1u,   // an mbarrier wait exceeded kWaitNs
    kErrStoreTimeout = 2u,  // reserved
    kErrPlan = 4u,          // a CTA's token share does not fit the launch's tile-group plan
};

constexpr unsigned long long kWaitNs = 2000000000ull;  // 2 s

__device__ __forceinline__ uint32_t smem_u32(const void *p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ unsigned long long globaltimer()
{
    unsigned long long t;
    asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
    return t;
}

// Programmatic dependent launch: wait until the previous kernel of the stream has completed and
// its memory is visible (a no-op when the launch had no programmatic dependency), and let the
// next kernel be scheduled now (it waits the same way before it touches memory).
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// Fetch the 128-byte line holding p into L2 (no register result, no wait).
__device__ __forceinline__ void prefetch_l2(const void *p)
{
    asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}

__device__ __forceinline__ void flag_error(unsigned code)
{
    atomicOr(&g_resbm_device_error, code);
}

// Token range [start, end) of CTA b out of G over T tokens: T is cut into whole 128-token
// tiles and every CTA gets a contiguous run of floor or ceil(tiles / G) of them; only the
// tensor's last tile can be partial. (A partial tile streams through as many pipeline stages as
// a full one and costs about as much time, so balancing to finer units made every CTA pay for
// one; with whole tiles the CTAs with one tile fewer finish early and leave the bandwidth to the
// others. The grid is at most the number of tiles.)
__device__ __forceinline__ void token_range(int64_t T, int b, int G, int64_t &start, int64_t &end)
{
    const int64_t U = (T + 127) / 128;
    start = 128 * ((U * b) / G);
    end = 128 * ((U * (b + 1)) / G);
    if (end > T) end = T;
    if (start > T) start = T;
}

// Tiles [tb, te) of tile group g when a CTA's ntiles tiles are cut into ngroups groups as evenly
// as possible, the larger groups first: the kernels' per-tile barriers (one per position in a
// group, waited with the group's parity) need every position used by a group to have been used
// by all earlier groups. Every CTA of a launch has the same ngroups (so that the CTAs of a
// cluster make the same sequence of weight-gradient exchanges); the host picks it so that every
// group has between 1 and the kernel's group capacity of tiles.
__device__ __forceinline__ void group_tiles(int g, int ngroups, int ntiles, int &tb, int &te)
{
    const int q = ntiles / ngroups, rem = ntiles - q * ngroups;
    tb = g * q + (g < rem ? g : rem);
    te = tb + q + (g < rem ? 1 : 0);
}

// ---- small per-token products on CUDA cores (fp32 accumulate) ---------------------------------
// acc[0..16) = sum over k of x[k] * W[k][n0 .. n0 + 16), W a K x N row-major bf16 matrix in
// shared memory (rows 16-byte aligned); k runs in order 0, 1, ..., K-1.
template <int K, int N>
__device__ __forceinline__ void vecmat16(const float (&x)[K], const __nv_bfloat16 *W, int n0, float (&acc)[16])
{
#pragma unroll
    for (int i = 0; i < 16; ++i) acc[i] = 0.0f;
#pragma unroll
    for (int k = 0; k < K; ++k) {
        const uint4 *w = reinterpret_cast<const uint4 *>(W + k * N + n0);
        const uint4 w0 = w[0], w1 = w[1];
        const uint32_t wv[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            acc[2 * j] = fmaf(x[k], __uint_as_float(wv[j] << 16), acc[2 * j]);
            acc[2 * j + 1] = fmaf(x[k], __uint_as_float(wv[j] & 0xFFFF0000u), acc[2 * j + 1]);
        }
    }
}

// A row of N bf16 values (16-byte aligned, N % 8 == 0) as fp32.
template <int N> __device__ __forceinline__ void load_bf16_row(const __nv_bfloat16 *src, float (&x)[N])
{
    const uint4 *s = reinterpret_cast<const uint4 *>(src);
#pragma unroll
    for (int v = 0; v < N / 8; ++v) {
        const uint4 u = s[v];
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            x[8 * v + 2 * e] = __uint_as_float(w[e] << 16);
            x[8 * v + 2 * e + 1] = __uint_as_float(w[e] & 0xFFFF0000u);
        }
    }
}

// ---- mbarrier ---------------------------------------------------------------------------------
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init()
{
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar)
{
    asm volatile("{\n\t.reg .b64 st;\n\tmbarrier.arrive.shared::cta.b64 st, [%0];\n\t}" ::"r"(bar)
                 : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes)
{
    asm volatile("{\n\t.reg .b64 st;\n\tmbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n\t}" ::"r"(bar),
                 "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Non-blocking test: has the phase with the given parity completed?
__device__ __forceinline__ bool mbar_test_wait(uint32_t bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Wait for the phase with the given parity to complete; false (and an error flag) on timeout.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity)
{
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = globaltimer();
    for (uint32_t i = 1;; ++i) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((i & 255u) == 0 && globaltimer() - t0 > kWaitNs) {
            flag_error(kErrWaitTimeout);
            return false;
        }
    }
}

// ---- thread-block clusters --------------------------------------------------------------------
__device__ __forceinline__ uint32_t cluster_rank()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

__device__ __forceinline__ uint32_t cluster_size()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
    return r;
}

__device__ __forceinline__ uint32_t cluster_index()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
    return r;
}

// The address of the same shared-memory location in cluster CTA `rank` (distributed shared memory).
__device__ __forceinline__ uint32_t map_shared(uint32_t addr, uint32_t rank)
{
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
    return r;
}

// All threads of all CTAs of the cluster (release / acquire at cluster scope).
__device__ __forceinline__ void cluster_sync()
{
    asm volatile("barrier.cluster.arrive;\n\tbarrier.cluster.wait;" ::: "memory");
}

// Arrive on an mbarrier of another CTA of the cluster (address from map_shared). Default
// semantics (release at CTA scope): used only to hand a shared-memory buffer back to its writer
// after the values read from it have been consumed, which needs no cluster-scope fence.
__device__ __forceinline__ void mbar_arrive_remote(uint32_t cluster_bar)
{
    asm volatile("mbarrier.arrive.shared::cluster.b64 _, [%0];" ::"r"(cluster_bar) : "memory");
}

// 16-byte store into another CTA's shared memory that counts its bytes on that CTA's mbarrier
// (both addresses from map_shared). The bytes are visible to the threads that see the barrier's
// phase complete, as with a TMA load.
__device__ __forceinline__ void st_async_f4(uint32_t cluster_dst, float4 v, uint32_t cluster_bar)
{
    asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.f32 [%0], {%1, %2, %3, %4}, [%5];" ::"r"(
                     cluster_dst),
                 "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w), "r"(cluster_bar)
                 : "memory");
}

// ---- proxies and fences -------------------------------------------------------------------------
// Make generic-proxy writes to shared memory visible to the async proxy (TMA, tensor cores).
__device__ __forceinline__ void fence_async_smem()
{
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void named_barrier(uint32_t id, uint32_t nthreads)
{
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

__device__ __forceinline__ bool elect_one()
{
    uint32_t pred = 0;
    asm volatile(
        "{\n\t.reg .pred p;\n\telect.sync _|p, 0xffffffff;\n\tselp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(pred));
    return pred != 0;
}

// ---- TMA ----------------------------------------------------------------------------------------
__device__ __forceinline__ void tma_prefetch_desc(const CUtensorMap *m)
{
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(m)) : "memory");
}

// 2D tiled load of the box at (x = inner element, y = row) into shared memory; completes
// `bytes` of transaction count on `bar`.
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *m, int32_t x, int32_t y,
                                            uint32_t bar)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(m)), "r"(x), "r"(y), "r"(bar)
        : "memory");
}

// 2D tiled store of a shared-memory box to (x, y); rows/columns outside the tensor are skipped.
// L2 cache policies: data streamed through once goes first when L2 must evict; data that is read
// back soon (the weight-gradient partial slots) goes last.
__device__ __forceinline__ uint64_t l2_evict_first()
{
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}
__device__ __forceinline__ uint64_t l2_evict_last()
{
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
    return p;
}

// tma_load_2d with an L2 cache policy
__device__ __forceinline__ void tma_load_2d_hint(uint32_t dst, const CUtensorMap *m, int32_t x, int32_t y,
                                                 uint32_t bar, uint64_t policy)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(m)), "r"(x), "r"(y), "r"(bar), "l"(policy)
        : "memory");
}

// tma_store_2d with an L2 cache policy
__device__ __forceinline__ void tma_store_2d_hint(const CUtensorMap *m, int32_t x, int32_t y, uint32_t src,
                                                  uint64_t policy)
{
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.tile.bulk_group.L2::cache_hint [%0, {%1, %2}], [%3], %4;" ::"l"(
                     reinterpret_cast<uint64_t>(m)),
                 "r"(x), "r"(y), "r"(src), "l"(policy)
                 : "memory");
}

// 16-byte global store with an L2 cache policy
__device__ __forceinline__ void st_global_hint(float4 *p, float4 v, uint64_t policy)
{
    asm volatile("st.global.L2::cache_hint.v4.f32 [%0], {%1, %2, %3, %4}, %5;" ::"l"(p), "f"(v.x), "f"(v.y),
                 "f"(v.z), "f"(v.w), "l"(policy)
                 : "memory");
}

__device__ __forceinline__ void tma_store_2d(const CUtensorMap *m, int32_t x, int32_t y, uint32_t src)
{
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.tile.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
                     reinterpret_cast<uint64_t>(m)),
                 "r"(x), "r"(y), "r"(src)
                 : "memory");
}

__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }

// Wait until at most N committed store groups still read shared memory.
template <int N> __device__ __forceinline__ void bulk_wait_read()
{
    asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}

template <int N> __device__ __forceinline__ void bulk_wait()
{
    asm volatile("cp.async.bulk.wait_group %0;" ::"n"(N) : "memory");
}

// ---- tcgen05: tensor memory -----------------------------------------------------------------------
// Allocate ncols (power of two >= 32) TMEM columns; executed by one whole warp. The base address
// is written to shared memory at `dst`.
__device__ __forceinline__ void tmem_alloc(uint32_t dst, uint32_t ncols)
{
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst), "r"(ncols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols)
{
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// D[tmem] (+)= A[smem desc] * B[smem desc], kind::f16 (bf16 inputs, fp32 accumulate), one CTA.
__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                         bool accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a_desc), "l"(b_desc), "r"(idesc), "r"((uint32_t)accumulate)
        : "memory");
}

// Arrive once on `bar` when every MMA issued so far by this thread has completed.
__device__ __forceinline__ void mma_commit(uint32_t bar)
{
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}

// Each thread of the warp reads 32 consecutive fp32 columns of its own TMEM lane
// (lane = the warp's 32-lane quarter + lane id); taddr = (quarter base lane << 16) | column.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32])
{
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, "
        "%13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, "
        "[%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
          "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
          "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]),
          "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16])
{
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, "
        "%13, %14, %15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
          "=r"(r[15])
        : "r"(taddr));
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// After tmem_ld_wait: ties the loaded registers to that point, so that no use of them can be
// scheduled above the wait (the loads write them asynchronously until it).
template <int N> __device__ __forceinline__ void tmem_regs_ready(float (&v)[N])
{
#pragma unroll
    for (int i = 0; i < N; ++i) asm volatile("" : "+f"(v[i]));
}

// ---- descriptors --------------------------------------------------------------------------------
// Swizzle modes of the shared-memory matrix descriptor (bits 61..63) and their row widths.
enum Swz : uint32_t { kSwzNone = 0, kSwz128 = 2, kSwz64 = 4, kSwz32 = 6 };

__host__ __device__ constexpr uint32_t swz_bytes(Swz s)
{
    return s == kSwz128 ? 128u : s == kSwz64 ? 64u : s == kSwz32 ? 32u : 16u;
}

// Shared-memory matrix descriptor (tcgen05): start address, leading- and stride-dimension byte
// offsets (all >> 4), descriptor version 1 (bit 46), swizzle mode. For K-major swizzled operands
// SBO is the distance between 8-row groups (LBO unused); for MN-major swizzled operands LBO is the
// distance between swizzle-wide blocks along M/N and SBO the distance between 8-row groups along K.
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr, uint32_t lbo, uint32_t sbo, Swz swz)
{
    uint64_t d = 0;
    d |= (uint64_t)((addr >> 4) & 0x3FFFu);
    d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
    d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
    d |= 1ull << 46;
    d |= (uint64_t)swz << 61;
    return d;
}

// Descriptor increment (bytes >> 4) of K step k (16 bf16 elements) inside a K-major operand of
// 128-byte swizzled 64-column blocks: 4 steps of 32 bytes per block, blocks `block_bytes` apart.
__host__ __device__ constexpr uint64_t kmaj_off(int k, uint32_t block_bytes)
{
    return (uint64_t)(((uint32_t)(k >> 2) * block_bytes + (uint32_t)(k & 3) * 32u) >> 4);
}

// Instruction descriptor for kind::f16 with bf16 A and B, fp32 D, dense, M x N.
// a_mn / b_mn: operand stored MN-major (transposed) instead of K-major.
__host__ __device__ constexpr uint32_t idesc_bf16(uint32_t M, uint32_t N, bool a_mn, bool b_mn)
{
    return (1u << 4)                 // D format: f32
           | (1u << 7)               // A format: bf16
           | (1u << 10)              // B format: bf16
           | ((a_mn ? 1u : 0u) << 15) | ((b_mn ? 1u : 0u) << 16) | ((N >> 3) << 17) | ((M >> 4) << 24);
}

// Byte offset of element (row, col) of a swizzled tile whose rows are `swz_bytes` wide
// (16-byte chunk index XOR row % 8, the TMA / UMMA swizzle pattern); tile base 1024-B aligned.
__device__ __forceinline__ uint32_t swz_offset(uint32_t row, uint32_t byte_in_row, uint32_t row_bytes)
{
    const uint32_t chunk = byte_in_row >> 4;
    const uint32_t mask = row_bytes == 128 ? 7u : row_bytes == 64 ? 3u : row_bytes == 32 ? 1u : 0u;
    // 128B: chunk ^= row % 8; 64B: chunk ^= (row / 2) % 4; 32B: chunk ^= (row / 4) % 2
    const uint32_t sel = row_bytes == 128 ? (row & 7u) : row_bytes == 64 ? ((row >> 1) & 3u)
                                                                          : ((row >> 2) & 1u);
    return row * row_bytes + (((chunk ^ sel) & mask) << 4) + (byte_in_row & 15u);
}

// The N (a multiple of 16) fp32 TMEM columns at taddr of this thread's lane (warp-collective).
template <int N> __device__ __forceinline__ void tmem_ld_row(uint32_t taddr, float (&v)[N])
{
#pragma unroll
    for (int j = 0; j < N; j += 16) {
        float t[16];
        tmem_ld16(taddr + j, t);
        tmem_ld_wait();
#pragma unroll
        for (int e = 0; e < 16; ++e) v[j + e] = t[e];
    }
}

// Row `row` of a swizzled bf16 tile whose rows are N elements (2N bytes, the swizzle width):
// store N fp32 values rounded to bf16, or load them back as fp32 (16-byte accesses).
template <int N> __device__ __forceinline__ void store_bf16_swz_row(uint8_t *tile, int row, const float (&v)[N])
{
#pragma unroll
    for (int cc = 0; cc < N / 8; ++cc) {
        uint32_t pk[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            __nv_bfloat162 h = __floats2bfloat162_rn(v[8 * cc + 2 * e], v[8 * cc + 2 * e + 1]);
            pk[e] = *reinterpret_cast<uint32_t *>(&h);
        }
        *reinterpret_cast<uint4 *>(tile + swz_offset(row, 16 * cc, 2 * N)) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
    }
}

template <int N> __device__ __forceinline__ void load_bf16_swz_row(const uint8_t *tile, int row, float (&v)[N])
{
#pragma unroll
    for (int cc = 0; cc < N / 8; ++cc) {
        const uint4 u = *reinterpret_cast<const uint4 *>(tile + swz_offset(row, 16 * cc, 2 * N));
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            v[8 * cc + 2 * e] = __uint_as_float(w[e] << 16);
            v[8 * cc + 2 * e + 1] = __uint_as_float(w[e] & 0xFFFF0000u);
        }
    }
}

// Swizzle mode of a K-major or MN-major operand whose rows are `row_bytes` (32, 64 or 128).
__host__ __device__ constexpr Swz swz_for(uint32_t row_bytes)
{
    return row_bytes == 128 ? kSwz128 : row_bytes == 64 ? kSwz64 : kSwz32;
}

}  // namespace tc
}  // namespace resbm
