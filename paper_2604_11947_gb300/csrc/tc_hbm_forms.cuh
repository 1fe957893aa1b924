// tc_hbm_forms.cuh -- the HBM rate each access form attains on this device, measured with the
// forms the boundary kernels use and the ones they were weighed against:
//   plain 16-byte loads, stores and copies by every thread of four 512-thread CTAs per SM;
//   one CTA per SM streaming through a ring of 128 KB of shared-memory stages with
//     2-D tensor loads of 64-column x 128-row bf16 boxes (16 KB, 128-byte swizzle), one box or
//     two boxes per stage, or one 3-D box of two such column blocks per stage,
//     1-D bulk copies of 16 KB,
//     2-D tensor stores of the same boxes, and 1-D bulk stores of 16 KB;
//   and the 2-D loads and stores in the backward kernels' walk (below).
// Not a step of the method: a measurement of the memory system that the kernels' choice of load
// and store forms and of their ring depths rests on. The TMA forms view a buffer as a row-major
// bf16 matrix of 4096 columns (8 KB rows, the boundary tensors' rows at d = 4096); every CTA
// takes a contiguous run of boxes, in row-tile-major order (each 128-row tile, 1 MB of
// contiguous memory, box after box), or in the walk of the backward kernels: its run of 128-row
// tiles in groups of up to four, and per group the 128-column chunks in cyclic order from a
// chunk that depends on the CTA, each chunk's tiles one after the other (two boxes per tile).
#pragma once

#include "tc_common.cuh"

namespace resbm {
namespace tc {

constexpr uint32_t kFormBox = 16384;          // one 64 x 128 bf16 box
constexpr int kFormBlocks = 64;               // 64-column blocks per 8 KB row
constexpr int kFormRingBoxes = 8;             // 128 KB in flight per CTA
constexpr uint32_t kFormSmem = kFormRingBoxes * kFormBox + 1024;

// forms of k_form_load
constexpr int kLoad2d = 0, kLoad2dPair = 1, kLoad3d = 2, kLoadBulk = 3, kLoadTiles = 4;
// forms of k_form_store
constexpr int kStore2d = 0, kStoreBulk = 1, kStoreTiles = 2;

// The backward kernels' walk: the q-th (tile, chunk) pair of a CTA whose run is the 128-row
// tiles [t0, t1), in groups of up to 4 tiles, chunks from c_first on. Returns x (column) and y (row).
__device__ __forceinline__ void tiles_walk(int64_t q, int64_t t0, int64_t t1, int c_first, int32_t &x, int32_t &y)
{
    constexpr int NC = kFormBlocks / 2;   // 128-column chunks per row
    const int64_t g0 = t0 + 4 * (q / (4 * NC));
    const int64_t gsz = t1 - g0 < 4 ? t1 - g0 : 4;   // only the last group can be short
    const int64_t w = q % (4 * NC);
    const int c = (int)((w / gsz + c_first) % NC);
    x = c * 128;
    y = (int32_t)((g0 + w % gsz) * 128);
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap *m, int32_t x, int32_t y, int32_t z,
                                            uint32_t bar)
{
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(m)), "r"(x), "r"(y), "r"(z), "r"(bar)
        : "memory");
}

// 1-D bulk copy of `bytes` contiguous bytes (16-byte aligned, a multiple of 16) into shared memory
__device__ __forceinline__ void bulk_load(uint32_t dst, const void *src, uint32_t bytes, uint32_t bar)
{
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
                 "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(bar)
                 : "memory");
}

// 1-D bulk copy of `bytes` contiguous bytes from shared memory to global memory (a bulk group)
__device__ __forceinline__ void bulk_store(void *dst, uint32_t src, uint32_t bytes)
{
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(reinterpret_cast<uint64_t>(dst)),
                 "r"(src), "r"(bytes)
                 : "memory");
}

// One elected thread per CTA streams its run of the buffer's boxes through the ring; nothing
// reads the landed bytes (the rate of the loads alone). `boxes` = the buffer's 16 KB boxes, a
// multiple of kFormBlocks (whole 128-row tiles).
template <int FORM>
__global__ void __launch_bounds__(128, 1)
    k_form_load(const __grid_constant__ CUtensorMap map, const uint8_t *src, int64_t boxes)
{
    // boxes per stage
    constexpr int PER = (FORM == kLoad2dPair || FORM == kLoad3d || FORM == kLoadTiles) ? 2 : 1;
    constexpr int NST = kFormRingBoxes / PER;
    constexpr uint32_t STAGE = PER * kFormBox;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    __shared__ uint64_t full[NST];
    if (threadIdx.x == 0) {
        for (int s = 0; s < NST; ++s) mbar_init(smem_u32(&full[s]), 1);
        fence_mbar_init();
    }
    __syncthreads();
    if (threadIdx.x != 0) return;
    if (FORM != kLoadBulk) tma_prefetch_desc(&map);
    const int64_t n = boxes / PER;   // stages over the whole buffer
    int64_t b = n * blockIdx.x / gridDim.x, e = n * (blockIdx.x + 1) / gridDim.x;
    const int64_t tiles = boxes / kFormBlocks;
    const int64_t t0 = tiles * blockIdx.x / gridDim.x, t1 = tiles * (blockIdx.x + 1) / gridDim.x;
    if (FORM == kLoadTiles) {   // whole tiles per CTA: 32 stages each
        b = t0 * (kFormBlocks / 2);
        e = t1 * (kFormBlocks / 2);
    }
    int64_t k = 0;   // stages issued by this CTA
    for (int64_t v = b; v < e; ++v, ++k) {
        const int s = (int)(k % NST);
        // the stage's previous fill (issue k - NST) has landed
        if (k >= NST && !mbar_wait(smem_u32(&full[s]), (uint32_t)((k / NST - 1) & 1))) break;
        const uint32_t bar = smem_u32(&full[s]);
        const uint32_t dst = smem_u32(smem + s * STAGE);
        mbar_expect_tx(bar, STAGE);
        if (FORM == kLoad2d) {
            tma_load_2d(dst, &map, (int32_t)(v % kFormBlocks) * 64, (int32_t)(v / kFormBlocks) * 128, bar);
        } else if (FORM == kLoad2dPair) {
            const int32_t x = (int32_t)(v % (kFormBlocks / 2)) * 128, y = (int32_t)(v / (kFormBlocks / 2)) * 128;
            tma_load_2d(dst, &map, x, y, bar);
            tma_load_2d(dst + kFormBox, &map, x + 64, y, bar);
        } else if (FORM == kLoadTiles) {
            int32_t x, y;
            tiles_walk(v - b, t0, t1, (int)(blockIdx.x % (kFormBlocks / 2)), x, y);
            tma_load_2d(dst, &map, x, y, bar);
            tma_load_2d(dst + kFormBox, &map, x + 64, y, bar);
        } else if (FORM == kLoad3d) {
            tma_load_3d(dst, &map, 0, (int32_t)(v / (kFormBlocks / 2)) * 128, (int32_t)(v % (kFormBlocks / 2)) * 2, bar);
        } else {
            bulk_load(dst, src + v * (int64_t)kFormBox, kFormBox, bar);
        }
    }
    // the stages still in flight land before the CTA exits
    for (int64_t j = k > NST ? k - NST : 0; j < k; ++j) mbar_wait(smem_u32(&full[j % NST]), (uint32_t)((j / NST) & 1));
}

// One elected thread per CTA writes its run of the buffer's boxes from the ring of staging
// boxes (every byte 0xA5), at most kFormRingBoxes stores reading shared memory at a time.
template <int FORM>
__global__ void __launch_bounds__(128, 1)
    k_form_store(const __grid_constant__ CUtensorMap map, uint8_t *dst, int64_t boxes)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    for (uint32_t i = threadIdx.x; i < kFormRingBoxes * kFormBox / 16; i += blockDim.x)
        reinterpret_cast<uint4 *>(smem)[i] = make_uint4(0xA5A5A5A5u, 0xA5A5A5A5u, 0xA5A5A5A5u, 0xA5A5A5A5u);
    fence_async_smem();
    __syncthreads();
    if (threadIdx.x != 0) return;
    if (FORM != kStoreBulk) tma_prefetch_desc(&map);
    int64_t b = boxes * blockIdx.x / gridDim.x, e = boxes * (blockIdx.x + 1) / gridDim.x;
    const int64_t tiles = boxes / kFormBlocks;
    const int64_t t0 = tiles * blockIdx.x / gridDim.x, t1 = tiles * (blockIdx.x + 1) / gridDim.x;
    if (FORM == kStoreTiles) {   // whole tiles per CTA: 64 boxes each
        b = t0 * kFormBlocks;
        e = t1 * kFormBlocks;
    }
    int64_t k = 0;
    for (int64_t v = b; v < e; ++v, ++k) {
        if (k >= kFormRingBoxes) bulk_wait_read<kFormRingBoxes - 1>();   // store k - 8 has read its box
        const uint32_t src = smem_u32(smem + (uint32_t)(k % kFormRingBoxes) * kFormBox);
        if (FORM == kStore2d) {
            tma_store_2d(&map, (int32_t)(v % kFormBlocks) * 64, (int32_t)(v / kFormBlocks) * 128, src);
        } else if (FORM == kStoreTiles) {   // the tile's two 64-column halves of a chunk in turn
            int32_t x, y;
            tiles_walk((v - b) / 2, t0, t1, (int)(blockIdx.x % (kFormBlocks / 2)), x, y);
            tma_store_2d(&map, x + 64 * (int32_t)((v - b) & 1), y, src);
        } else {
            bulk_store(dst + v * (int64_t)kFormBox, src, kFormBox);
        }
        bulk_commit();
    }
    bulk_wait<0>();
}

// Plain 16-byte accesses, four in flight per thread, four CTAs of 512 threads per SM. The loads
// fold into a word that is written out only if it equals a constant no input is expected to
// produce, which keeps them.
__global__ void __launch_bounds__(512, 4) k_form_read_v4(const uint4 *p, int64_t n, unsigned *sink)
{
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    unsigned acc = 0;
#pragma unroll 1
    for (; i + 3 * stride < n; i += 4 * stride) {
        const uint4 a = __ldcs(p + i), b = __ldcs(p + i + stride), c = __ldcs(p + i + 2 * stride),
                    d = __ldcs(p + i + 3 * stride);
        acc ^= (a.x ^ a.y ^ a.z ^ a.w) ^ (b.x ^ b.y ^ b.z ^ b.w) ^ (c.x ^ c.y ^ c.z ^ c.w) ^ (d.x ^ d.y ^ d.z ^ d.w);
    }
#pragma unroll 1
    for (; i < n; i += stride) {
        const uint4 a = __ldcs(p + i);
        acc ^= a.x ^ a.y ^ a.z ^ a.w;
    }
    if (acc == 0x9E3779B9u) *sink = acc;
}

__global__ void __launch_bounds__(512, 4) k_form_write_v4(uint4 *p, int64_t n)
{
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const uint4 v = make_uint4(0xA5A5A5A5u, 0xA5A5A5A5u, 0xA5A5A5A5u, 0xA5A5A5A5u);
#pragma unroll 4
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) p[i] = v;
}

__global__ void __launch_bounds__(512, 4) k_form_copy_v4(const uint4 *s, uint4 *d, int64_t n)
{
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
#pragma unroll 1
    for (; i + 3 * stride < n; i += 4 * stride) {
        const uint4 a = __ldcs(s + i), b = __ldcs(s + i + stride), c = __ldcs(s + i + 2 * stride),
                    e = __ldcs(s + i + 3 * stride);
        d[i] = a;
        d[i + stride] = b;
        d[i + 2 * stride] = c;
        d[i + 3 * stride] = e;
    }
#pragma unroll 1
    for (; i < n; i += stride) d[i] = __ldcs(s + i);
}

}  // namespace tc
}  // namespace resbm
