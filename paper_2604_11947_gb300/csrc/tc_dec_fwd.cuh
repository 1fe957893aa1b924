// tc_dec_fwd.cuh -- receive side of the boundary on tensor cores (Sec. 3.2 decoder, Eq. Pid
// zero-padding identity path):  Y = [merge] B . I_{r x d} + phi(B . Wd1) . Wd2.
//
// Persistent CTAs; CTA b owns a contiguous token range (16-token aligned, balanced to within
// 16 tokens) and walks it in tiles of up to 128 tokens. Per tile:
//   epilogue warps : Q = B . Wd1 on CUDA cores (fp32), G = phi(Q) -> bf16 -> shared memory
//                    (the MMA A operand, K-major, 128B swizzle)
//   producer warp  : Wd2 column chunks (m x NCH, MN-major B operand) by TMA into a ring
//   MMA warp       : D_chunk (128 x NCH fp32, TMEM, double-buffered) = G . Wd2_chunk
//   epilogue warps : TMEM -> registers, + B on the first r columns, -> bf16 -> swizzled staging
//                    -> TMA store of Y (boxes of 128 rows, or 16 rows for a partial tile)
// HBM traffic per token: read B (2r bytes), write Y (2d bytes); Wd2 is re-read from L2.
#pragma once

#include "common.cuh"
#include "tc_common.cuh"

namespace resbm {
namespace tc {

template <int M_> struct DecFwdCfg {
    static constexpr int M = M_;                       // hidden width m (= r on this path)
    static constexpr int R = M_;                       // bottleneck width r
    static constexpr int NCH = M_ <= 32 ? 256 : 128;   // Y columns per MMA chunk
    static constexpr int NSTAGE = M_ <= 64 ? 3 : 2;    // Wd2 chunk ring depth
    static constexpr int KBLK = (M_ + 63) / 64;        // 64-wide K blocks of G
    static constexpr uint32_t W_STAGE_BYTES = M_ * NCH * 2;
    static constexpr uint32_t G_BYTES = KBLK * 128 * 128;
    static constexpr uint32_t STG_BYTES = 128 * NCH * 2;
    static constexpr uint32_t WD1_BYTES = R * M_ * 2;
    // shared-memory map (offsets from a 1024-aligned base)
    static constexpr uint32_t OFF_W = 0;
    static constexpr uint32_t OFF_G = OFF_W + NSTAGE * W_STAGE_BYTES;
    static constexpr uint32_t OFF_STG = OFF_G + 2 * G_BYTES;
    static constexpr uint32_t OFF_WD1 = OFF_STG + 2 * STG_BYTES;
    static constexpr uint32_t SMEM_BYTES = OFF_WD1 + WD1_BYTES + 1024;  // + alignment slack
    static constexpr uint32_t TMEM_COLS = 2 * NCH;
    static constexpr int THREADS = 192;
};

struct DecFwdArgs {
    const __nv_bfloat16 *B;     // T x r
    const __nv_bfloat16 *Wd1;   // r x m
    int64_t T, d;
    int act, merge;
};

template <int M_>
__global__ void __launch_bounds__(192, 1)
    k_dec_fwd(const __grid_constant__ CUtensorMap tm_wd2, const __grid_constant__ CUtensorMap tm_y128,
              const __grid_constant__ CUtensorMap tm_y16, const DecFwdArgs a)
{
    using C = DecFwdCfg<M_>;
    griddep_wait();               // the previous kernel of the stream has completed
    griddep_launch_dependents();  // the next one may be scheduled on SMs as they free up
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    __shared__ uint64_t w_full[C::NSTAGE], w_empty[C::NSTAGE];
    __shared__ uint64_t g_full[2], g_empty[2], acc_full[2], acc_empty[2], done_bar;
    __shared__ uint32_t tmem_base_sh;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nchunks = (int)(a.d / C::NCH) + ((a.d % C::NCH) ? 1 : 0);
    int64_t start, end;
    token_range(a.T, blockIdx.x, gridDim.x, start, end);

    if (threadIdx.x == 0) {
        for (int s = 0; s < C::NSTAGE; ++s) {
            mbar_init(smem_u32(&w_full[s]), 1);
            mbar_init(smem_u32(&w_empty[s]), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(smem_u32(&g_full[i]), 1);
            mbar_init(smem_u32(&g_empty[i]), 1);
            mbar_init(smem_u32(&acc_full[i]), 1);
            mbar_init(smem_u32(&acc_empty[i]), 128);
        }
        mbar_init(smem_u32(&done_bar), 1);
        fence_mbar_init();
    }
    if (warp == 1) tmem_alloc(smem_u32(&tmem_base_sh), C::TMEM_COLS);
    if (warp >= 2) {  // Wd1 (r x m bf16) into shared memory, once
        const uint4 *src = reinterpret_cast<const uint4 *>(a.Wd1);
        uint4 *dst = reinterpret_cast<uint4 *>(smem + C::OFF_WD1);
        for (int i = threadIdx.x - 64; i < (int)(C::WD1_BYTES / 16); i += 128) dst[i] = src[i];
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_base_sh;

    if (warp == 0) {
        // ---------------- producer: Wd2 chunks ----------------
        if (elect_one()) {
            tma_prefetch_desc(&tm_wd2);
            uint32_t it = 0;
            bool ok = true;
            for (int64_t t0 = start; t0 < end && ok; t0 += 128) {
                for (int c = 0; c < nchunks; ++c) {
                    const uint32_t s = it % C::NSTAGE, ph = (it / C::NSTAGE) & 1;
                    if (!mbar_wait(smem_u32(&w_empty[s]), ph ^ 1)) {
                        ok = false;
                        break;
                    }
                    const uint32_t dst = smem_u32(smem + C::OFF_W + s * C::W_STAGE_BYTES);
                    mbar_expect_tx(smem_u32(&w_full[s]), C::W_STAGE_BYTES);
                    for (int b = 0; b < C::NCH / 64; ++b)
                        tma_load_2d(dst + b * (C::M * 128), &tm_wd2, c * C::NCH + 64 * b, 0, smem_u32(&w_full[s]));
                    ++it;
                }
            }
            // drain: every issued load has landed before the CTA can exit
            const uint32_t n = it < (uint32_t)C::NSTAGE ? it : (uint32_t)C::NSTAGE;
            for (uint32_t k = 0; k < n; ++k) {
                const uint32_t j = it - 1 - k;
                mbar_wait(smem_u32(&w_full[j % C::NSTAGE]), (j / C::NSTAGE) & 1);
            }
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if (elect_one()) {
            constexpr uint32_t idesc = idesc_bf16(128, C::NCH, false, true);
            uint32_t it = 0, acc_it = 0, tile_i = 0;
            bool ok = true;
            for (int64_t t0 = start; t0 < end && ok; t0 += 128, ++tile_i) {
                const uint32_t gb = tile_i & 1;
                ok = mbar_wait(smem_u32(&g_full[gb]), (tile_i >> 1) & 1);
                tc_fence_after();
                const uint32_t gaddr = smem_u32(smem + C::OFF_G + gb * C::G_BYTES);
                for (int c = 0; c < nchunks && ok; ++c, ++it, ++acc_it) {
                    const uint32_t s = it % C::NSTAGE, ph = (it / C::NSTAGE) & 1;
                    const uint32_t ab = acc_it & 1;
                    ok = mbar_wait(smem_u32(&w_full[s]), ph) &&
                         mbar_wait(smem_u32(&acc_empty[ab]), ((acc_it >> 1) & 1) ^ 1);
                    tc_fence_after();
                    const uint32_t waddr = smem_u32(smem + C::OFF_W + s * C::W_STAGE_BYTES);
#pragma unroll
                    for (int k = 0; k < C::M / 16; ++k) {
                        const uint64_t ad = smem_desc(gaddr + (k / 4) * 16384 + (k % 4) * 32, 16, 1024, kSwz128);
                        const uint64_t bd = smem_desc(waddr + k * 16 * 128, C::M * 128, 1024, kSwz128);
                        mma_bf16(tmem + ab * C::NCH, ad, bd, idesc, k > 0);
                    }
                    mma_commit(smem_u32(&w_empty[s]));
                    mma_commit(smem_u32(&acc_full[ab]));
                }
                mma_commit(smem_u32(&g_empty[gb]));
            }
            mma_commit(smem_u32(&done_bar));
            mbar_wait(smem_u32(&done_bar), 0);
        }
    } else {
        // ---------------- epilogue warps (128 threads, TMEM lane quarter = warp % 4) ----------------
        const int q = warp & 3;
        const int row = q * 32 + lane;
        const int et = threadIdx.x - 64;  // 0..127
        const __nv_bfloat16 *wd1 = reinterpret_cast<const __nv_bfloat16 *>(smem + C::OFF_WD1);
        uint32_t acc_it = 0, tile_i = 0, store_it = 0;
        bool ok = true;
        for (int64_t t0 = start; t0 < end && ok; t0 += 128, ++tile_i) {
            const int64_t t1 = (end - t0) < 128 ? end : t0 + 128;
            const int valid = (int)(t1 - t0);
            const bool active = row < valid;
            const int64_t tok = t0 + row;
            // B row (r bf16) in registers
            uint32_t brow[C::R / 2];
            if (active) {
                const uint4 *src = reinterpret_cast<const uint4 *>(a.B + tok * C::R);
#pragma unroll
                for (int i = 0; i < C::R / 8; ++i) {
                    const uint4 v = src[i];
                    brow[4 * i] = v.x; brow[4 * i + 1] = v.y; brow[4 * i + 2] = v.z; brow[4 * i + 3] = v.w;
                }
            } else {
#pragma unroll
                for (int i = 0; i < C::R / 2; ++i) brow[i] = 0u;
            }
            // G = phi(B . Wd1) -> bf16 -> G buffer (row `row`, K-major, 128B swizzle)
            const uint32_t gb = tile_i & 1;
            ok = mbar_wait(smem_u32(&g_empty[gb]), ((tile_i >> 1) & 1) ^ 1);
            uint8_t *gbuf = smem + C::OFF_G + gb * C::G_BYTES;
            // rows past the valid tokens only feed output rows that are never stored
            const int jend = (q * 32 < valid) ? C::M : 0;
#pragma unroll
            for (int jb = 0; jb < C::M; jb += 16) {
                if (jb >= jend) break;
                float accq[16];
#pragma unroll
                for (int j = 0; j < 16; ++j) accq[j] = 0.0f;
#pragma unroll
                for (int k = 0; k < C::R; ++k) {
                    const uint32_t bb = brow[k >> 1];
                    const float bk = __uint_as_float((k & 1) ? (bb & 0xFFFF0000u) : (bb << 16));
                    const uint4 *w = reinterpret_cast<const uint4 *>(wd1 + k * C::M + jb);
                    const uint4 w0 = w[0], w1 = w[1];
                    const uint32_t wv[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        accq[2 * j] = fmaf(bk, __uint_as_float(wv[j] << 16), accq[2 * j]);
                        accq[2 * j + 1] = fmaf(bk, __uint_as_float(wv[j] & 0xFFFF0000u), accq[2 * j + 1]);
                    }
                }
                act_fast_row<16>(a.act, accq);
                uint32_t packed[8];
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const float g0 = active ? accq[2 * j] : 0.0f;
                    const float g1 = active ? accq[2 * j + 1] : 0.0f;
                    __nv_bfloat162 h = __floats2bfloat162_rn(g0, g1);
                    packed[j] = *reinterpret_cast<uint32_t *>(&h);
                }
                // 16 bf16 = two 16-byte chunks at K offset jb within block jb / 64
                const uint32_t kb = jb >> 6, byte = (jb & 63) * 2;
                uint8_t *blk = gbuf + kb * 16384;
                *reinterpret_cast<uint4 *>(blk + swz_offset(row, byte, 128)) =
                    make_uint4(packed[0], packed[1], packed[2], packed[3]);
                *reinterpret_cast<uint4 *>(blk + swz_offset(row, byte + 16, 128)) =
                    make_uint4(packed[4], packed[5], packed[6], packed[7]);
            }
            fence_async_smem();
            named_barrier(1, 128);
            if (et == 0) mbar_arrive(smem_u32(&g_full[gb]));

            for (int c = 0; c < nchunks && ok; ++c, ++acc_it, ++store_it) {
                const uint32_t ab = acc_it & 1;
                const uint32_t sb = store_it & 1;
                ok = mbar_wait(smem_u32(&acc_full[ab]), (acc_it >> 1) & 1);
                tc_fence_after();
                if (et == 0) bulk_wait_read<1>();  // staging buffer sb is free again
                named_barrier(1, 128);
                uint8_t *stg = smem + C::OFF_STG + sb * C::STG_BYTES;
                const int64_t left = a.d - (int64_t)c * C::NCH;
                const int ncols = left < C::NCH ? (int)left : C::NCH;
                // a warp whose 32 rows all lie past the tile's valid tokens has nothing to store
                const int gend = (q * 32 < valid) ? ncols : 0;
#pragma unroll
                for (int g = 0; g < C::NCH / 32; ++g) {
                    if (g * 32 >= gend) break;
                    float v[32];
                    tmem_ld32(tmem + ((uint32_t)(q * 32) << 16) + ab * C::NCH + g * 32, v);
                    tmem_ld_wait();
                    // identity path: the first r columns of Y get B (only chunk 0 holds them)
                    if (g * 32 < C::R && a.merge && c == 0) {
#pragma unroll
                        for (int i = 0; i < 32; ++i) {
                            if (g * 32 + i < C::R) {
                                const uint32_t bb = brow[(g * 32 + i) >> 1];
                                v[i] += __uint_as_float(((g * 32 + i) & 1) ? (bb & 0xFFFF0000u) : (bb << 16));
                            }
                        }
                    }
                    uint32_t p[16];
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        __nv_bfloat162 h = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
                        p[i] = *reinterpret_cast<uint32_t *>(&h);
                    }
                    // columns [g*32, g*32+32) of the chunk: box g/2, bytes (g%2)*64 .. +64
                    uint8_t *box = stg + (g >> 1) * 16384;
                    const uint32_t b0 = (g & 1) * 64;
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        *reinterpret_cast<uint4 *>(box + swz_offset(row, b0 + 16 * i, 128)) =
                            make_uint4(p[4 * i], p[4 * i + 1], p[4 * i + 2], p[4 * i + 3]);
                }
                tc_fence_before();
                mbar_arrive(smem_u32(&acc_empty[ab]));
                fence_async_smem();
                named_barrier(1, 128);
                if (et == 0) {
                    const uint32_t sbase = smem_u32(stg);
                    for (int b = 0; b < ncols / 64; ++b) {
                        const int x = c * C::NCH + 64 * b;
                        if (valid == 128) {
                            tma_store_2d(&tm_y128, x, (int32_t)t0, sbase + b * 16384);
                        } else {
                            for (int rg = 0; rg * 16 < valid; ++rg)
                                tma_store_2d(&tm_y16, x, (int32_t)(t0 + 16 * rg), sbase + b * 16384 + rg * 2048);
                        }
                    }
                    bulk_commit();
                }
            }
        }
        if (et == 0) bulk_wait<0>();
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, C::TMEM_COLS);
    }
}

}  // namespace tc
}  // namespace resbm
