// tc_enc_bwd.cuh -- backward of the send side on tensor cores (chain rule of Sec. 3.2's encoder
// with the truncating identity path of Eq. Pid):
//   dP = (dB . We2^T) * phi'(P);  dF = dP . We1^T;  dX[:, :r] += dB;
//   dWe1 = F^T . dP;  dWe2 = phi(P)^T . dB.
//
// Persistent CTAs over contiguous 16-token-aligned token ranges, in groups of up to NT tiles.
//   phase 0 (epilogue warps): dP per token on CUDA cores (P from the forward pass), stored as
//            bf16 twice: rows = tokens (K-major over m; A operand of the dF product) and rows = m
//            (K-major over tokens; B operand of the dWe1 product). dX[:, :r] += dB.
//   phase 1 (producer + MMA): d in chunks of 128 columns; per chunk one We1 slice (128 x m,
//            K-major) and per tile one F tile (128 tokens x 128 columns) feeding
//              dF_tile_chunk (128 x 128 fp32, TMEM, double-buffered) = dP . We1_chunk^T
//              dWe1_chunk    (128 columns x m, TMEM, double-buffered) += F^T . dP
//            (F read as an MN-major operand). The epilogue converts dF to bf16 and stores it by
//            TMA, and drains each finished dWe1 chunk to the group's fp32 partial slot.
//   phase 3 (epilogue warps): the dWe2 partial (phi(P)^T . dB over the group's tokens, fixed
//            order) with the then idle F ring as scratch.
// HBM traffic per token: read F (2d), P (4m), dB (2r), dX[:, :r] (2r); write dF (2d), dX[:, :r]
// (2r); P and dB are read again in phase 3 (L2). Per slot: d x m + m x r fp32 partials.
#pragma once

#include "common.cuh"
#include "tc_common.cuh"
#include "tc_wgrad.cuh"

namespace resbm {
namespace tc {

template <int M_> struct EncBwdCfg {
    static constexpr int M = M_;
    static constexpr int R = M_;
    static constexpr int MS = M_ < 32 ? 32 : M_;                 // TMEM columns per dWe1 accumulator
    static constexpr int NT = M_ <= 32 ? 4 : 2;                  // tiles per group
    static constexpr int NSF = M_ <= 32 ? 3 : 2;                 // F ring depth
    static constexpr uint32_t DSW = M_ * 2 >= 128 ? 128 : M_ * 2;  // row bytes (= swizzle) of dP_A, We1
    static constexpr uint32_t F_STAGE = 128 * 128 * 2;
    static constexpr uint32_t STG_HALF = 128 * 64 * 2;           // dF staging: 128 rows x 64 columns
    static constexpr uint32_t W_STAGE = 128 * DSW;               // We1 slice: 128 rows x m
    static constexpr uint32_t DPA_TILE = 128 * DSW;              // dP, rows = tokens
    static constexpr uint32_t DPT_TILE = M_ * 256;               // dP^T, rows = m, 128 tokens
    static constexpr uint32_t WE2T_BYTES = R * M_ * 2;
    static constexpr uint32_t OFF_F = 0;
    static constexpr uint32_t OFF_STG = OFF_F + NSF * F_STAGE;
    static constexpr uint32_t OFF_W = OFF_STG + 2 * STG_HALF;
    static constexpr int NW = M_ <= 16 ? 4 : 3;                  // We1 slice ring depth
    static constexpr uint32_t OFF_DPA = OFF_W + NW * W_STAGE;
    static constexpr uint32_t OFF_DPT = OFF_DPA + NT * DPA_TILE;
    static constexpr uint32_t OFF_WE2T = OFF_DPT + NT * DPT_TILE;
    static constexpr uint32_t SMEM_BYTES = OFF_WE2T + WE2T_BYTES + 1024;
    static constexpr uint32_t SCRATCH_BYTES = 128 * (M_ + 1 + R + 1) * 4;  // phase 3: F ring + staging
    static_assert(SCRATCH_BYTES <= OFF_W, "phase-3 scratch must fit in the F ring and staging");
    static constexpr uint32_t TMEM_COLS = 512;                   // dF 2 x 128, dWe1 2 x MS
    static constexpr int THREADS = 192;
};

struct EncBwdArgs {
    const __nv_bfloat16 *dB;   // T x r
    const float *P;            // T x m
    const __nv_bfloat16 *We2;  // m x r
    __nv_bfloat16 *dX;         // T x d or null
    WgradArgs wg;              // dWe1 chunks (d x m), reduced across CTAs
    float *part2;              // slots x m x r  (dWe2 partials)
    int64_t T, d;
    int act, max_groups;
};

template <int M_>
__global__ void __launch_bounds__(192, 1)
    k_enc_bwd(const __grid_constant__ CUtensorMap tm_f128, const __grid_constant__ CUtensorMap tm_f16,
              const __grid_constant__ CUtensorMap tm_we1, const __grid_constant__ CUtensorMap tm_df128,
              const __grid_constant__ CUtensorMap tm_df16, const EncBwdArgs a)
{
    using C = EncBwdCfg<M_>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    __shared__ uint64_t f_full[C::NSF], f_empty[C::NSF], w_full[C::NW], w_empty[C::NW];
    __shared__ uint64_t dp_full[C::NT], dp_empty, df_full[2], df_empty[2], we_full[2], we_empty[2], p3_done, done_bar;
    __shared__ uint32_t tmem_base_sh;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nch = (int)(a.d / 128);
    int64_t start, end;
    token_range(a.T, blockIdx.x, gridDim.x, start, end);
    const int ntiles = (int)((end - start + 127) / 128);
    const int ngroups = (ntiles + C::NT - 1) / C::NT;

    if (threadIdx.x == 0) {
        for (int s = 0; s < C::NSF; ++s) {
            mbar_init(smem_u32(&f_full[s]), 1);
            mbar_init(smem_u32(&f_empty[s]), 1);
        }
        for (int i = 0; i < C::NW; ++i) {
            mbar_init(smem_u32(&w_full[i]), 1);
            mbar_init(smem_u32(&w_empty[i]), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(smem_u32(&df_full[i]), 1);
            mbar_init(smem_u32(&df_empty[i]), 128);
            mbar_init(smem_u32(&we_full[i]), 1);
            mbar_init(smem_u32(&we_empty[i]), 128);
        }
        for (int i = 0; i < C::NT; ++i) mbar_init(smem_u32(&dp_full[i]), 1);
        mbar_init(smem_u32(&dp_empty), 1);
        mbar_init(smem_u32(&p3_done), 1);
        mbar_init(smem_u32(&done_bar), 1);
        fence_mbar_init();
    }
    if (warp == 1) tmem_alloc(smem_u32(&tmem_base_sh), C::TMEM_COLS);
    if (warp >= 2) {  // We2^T (r x m bf16) into shared memory
        __nv_bfloat16 *dt = reinterpret_cast<__nv_bfloat16 *>(smem + C::OFF_WE2T);
        for (int e = threadIdx.x - 64; e < C::M * C::R; e += 128) dt[(e % C::R) * C::M + e / C::R] = a.We2[e];
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_base_sh;
    const uint32_t tmem_df = tmem;            // 2 x 128 columns
    const uint32_t tmem_we = tmem + 256;      // 2 x MS columns

    if (warp == 0) {
        // ---------------- producer ----------------
        if (elect_one()) {
            tma_prefetch_desc(&tm_f128);
            tma_prefetch_desc(&tm_f16);
            tma_prefetch_desc(&tm_we1);
            uint32_t fit = 0, wit = 0;
            bool ok = true;
            for (int g = 0; g < ngroups && ok; ++g) {
                if (g > 0) ok = mbar_wait(smem_u32(&p3_done), (g - 1) & 1);  // the ring was scratch
                const int tb = g * C::NT, te = min(ntiles, tb + C::NT);
                for (int c = 0; c < nch && ok; ++c) {
                    // order: F tile 0 of the chunk, the chunk's We1 slice, the other F tiles.
                    // The MMA needs the slice before any tile of the chunk, so it must not queue
                    // behind tiles that wait for ring slots (that would deadlock), and it must not
                    // delay the first tile (that would stall the stream on the small weight ring).
                    for (int i = tb; i < te; ++i) {
                        if (i == tb + 1) {
                            const uint32_t s = wit % C::NW;
                            if (!mbar_wait(smem_u32(&w_empty[s]), ((wit / C::NW) & 1) ^ 1)) { ok = false; break; }
                            mbar_expect_tx(smem_u32(&w_full[s]), C::W_STAGE);
                            tma_load_2d(smem_u32(smem + C::OFF_W + s * C::W_STAGE), &tm_we1, 0, c * 128,
                                        smem_u32(&w_full[s]));
                            ++wit;
                        }
                        const int64_t t0 = start + 128 * (int64_t)i;
                        const int valid = (int)((end - t0) < 128 ? (end - t0) : 128);
                        const int nb = (valid + 15) / 16;
                        const uint32_t s = fit % C::NSF;
                        if (!mbar_wait(smem_u32(&f_empty[s]), ((fit / C::NSF) & 1) ^ 1)) { ok = false; break; }
                        const uint32_t dst = smem_u32(smem + C::OFF_F + s * C::F_STAGE);
                        const uint32_t bar = smem_u32(&f_full[s]);
                        mbar_expect_tx(bar, valid == 128 ? C::F_STAGE : (uint32_t)nb * 2u * 2048u);
                        for (int h = 0; h < 2; ++h) {
                            if (valid == 128) {
                                tma_load_2d(dst + h * 16384, &tm_f128, c * 128 + 64 * h, (int32_t)t0, bar);
                            } else {
                                for (int rg = 0; rg < nb; ++rg)
                                    tma_load_2d(dst + h * 16384 + rg * 2048, &tm_f16, c * 128 + 64 * h,
                                                (int32_t)(t0 + 16 * rg), bar);
                            }
                        }
                        ++fit;
                    }
                    if (!ok) break;
                    if (te - tb == 1) {  // a one-tile group: the slice after its only tile
                        const uint32_t s = wit % C::NW;
                        if (!mbar_wait(smem_u32(&w_empty[s]), ((wit / C::NW) & 1) ^ 1)) { ok = false; break; }
                        mbar_expect_tx(smem_u32(&w_full[s]), C::W_STAGE);
                        tma_load_2d(smem_u32(smem + C::OFF_W + s * C::W_STAGE), &tm_we1, 0, c * 128,
                                    smem_u32(&w_full[s]));
                        ++wit;
                    }
                }
            }
            for (uint32_t k = 0; k < (fit < (uint32_t)C::NSF ? fit : (uint32_t)C::NSF); ++k) {
                const uint32_t j = fit - 1 - k;
                mbar_wait(smem_u32(&f_full[j % C::NSF]), (j / C::NSF) & 1);
            }
            for (uint32_t k = 0; k < (wit < (uint32_t)C::NW ? wit : (uint32_t)C::NW); ++k) {
                const uint32_t j = wit - 1 - k;
                mbar_wait(smem_u32(&w_full[j % C::NW]), (j / C::NW) & 1);
            }
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if (elect_one()) {
            constexpr Swz dswz = C::DSW == 128 ? kSwz128 : C::DSW == 64 ? kSwz64 : kSwz32;
            constexpr uint32_t id_df = idesc_bf16(128, 128, false, false);   // dP (K-major) . We1 (K-major)
            constexpr uint32_t id_we = idesc_bf16(128, C::M, true, false);   // F^T (MN-major) . dP^T (K-major)
            // shared-memory descriptors of slot / tile 0, advanced by adding byte offset >> 4 to
            // the start-address field (no carry: shared addresses < 256 KB)
            const uint64_t fm0 = smem_desc(smem_u32(smem + C::OFF_F), 16384, 1024, kSwz128);   // F, MN-major
            const uint64_t wd0 = smem_desc(smem_u32(smem + C::OFF_W), 16, 8 * C::DSW, dswz);   // We1 slice
            const uint64_t pa0 = smem_desc(smem_u32(smem + C::OFF_DPA), 16, 8 * C::DSW, dswz); // dP
            const uint64_t pt0 = smem_desc(smem_u32(smem + C::OFF_DPT), 16, 1024, kSwz128);    // dP^T
            uint32_t fit = 0, wit = 0, cit = 0, dfit = 0;
            bool ok = true;
            for (int g = 0; g < ngroups && ok; ++g) {
                const int tb = g * C::NT, te = min(ntiles, tb + C::NT);
                for (int c = 0; c < nch && ok; ++c, ++cit, ++wit) {
                    const uint32_t sw = wit % C::NW, ae = cit & 1;
                    ok = mbar_wait(smem_u32(&w_full[sw]), (wit / C::NW) & 1) &&
                         mbar_wait(smem_u32(&we_empty[ae]), ((cit >> 1) & 1) ^ 1);
                    tc_fence_after();
                    const uint64_t wd = wd0 + ((sw * C::W_STAGE) >> 4);
                    const uint32_t d_we = tmem_we + ae * C::MS;
                    for (int i = tb; i < te && ok; ++i, ++fit, ++dfit) {
                        const int64_t t0 = start + 128 * (int64_t)i;
                        const int valid = (int)((end - t0) < 128 ? (end - t0) : 128);
                        const uint32_t s = fit % C::NSF, ad_buf = dfit & 1;
                        // dP of the tile (phase 0, published per tile once per group), its F
                        // tile, a free dF buffer
                        if (c == 0) ok = mbar_wait(smem_u32(&dp_full[i - tb]), g & 1);
                        ok = ok && mbar_wait(smem_u32(&f_full[s]), (fit / C::NSF) & 1) &&
                             mbar_wait(smem_u32(&df_empty[ad_buf]), ((dfit >> 1) & 1) ^ 1);
                        tc_fence_after();
                        const uint64_t fm = fm0 + ((s * C::F_STAGE) >> 4);
                        const uint64_t pa = pa0 + (((i - tb) * C::DPA_TILE) >> 4);
                        const uint64_t pt = pt0 + (((i - tb) * C::DPT_TILE) >> 4);
                        const uint32_t d_df = tmem_df + ad_buf * 128;
                        // dF = dP . We1_chunk^T (K = m in steps of 16 = 32 bytes of a swizzled row)
#pragma unroll
                        for (int k = 0; k < C::M / 16; ++k) mma_bf16(d_df, pa + 2 * k, wd + 2 * k, id_df, k > 0);
                        mma_commit(smem_u32(&df_full[ad_buf]));
                        // dWe1^T_chunk += F^T . dP  (K = the tile's tokens in steps of 16)
                        if (valid == 128) {
#pragma unroll
                            for (int k = 0; k < 8; ++k)
                                mma_bf16(d_we, fm + ((k * 2048) >> 4), pt + kmaj_off(k, C::M * 128), id_we,
                                         (i > tb) || (k > 0));
                        } else {
                            const int nks = (valid + 15) / 16;
                            for (int k = 0; k < nks; ++k)
                                mma_bf16(d_we, fm + ((k * 2048) >> 4), pt + kmaj_off(k, C::M * 128), id_we,
                                         (i > tb) || (k > 0));
                        }
                        mma_commit(smem_u32(&f_empty[s]));
                    }
                    mma_commit(smem_u32(&w_empty[sw]));
                    mma_commit(smem_u32(&we_full[ae]));
                }
                mma_commit(smem_u32(&dp_empty));
            }
            mma_commit(smem_u32(&done_bar));
            mbar_wait(smem_u32(&done_bar), 0);
        }
    } else {
        // ---------------- epilogue warps ----------------
        const int q = warp & 3;
        const int row = q * 32 + lane;
        const int et = threadIdx.x - 64;
        const __nv_bfloat16 *we2t = reinterpret_cast<const __nv_bfloat16 *>(smem + C::OFF_WE2T);  // r x m
        constexpr int NOUT = (C::M * C::R + 127) / 128;
        uint32_t cit = 0, dfit = 0, sit = 0;
        bool ok = true;
        for (int g = 0; g < ngroups && ok; ++g) {
            const int tb = g * C::NT, te = min(ntiles, tb + C::NT);
            const int64_t slot = (int64_t)blockIdx.x * a.max_groups + g;
            // ---- phase 0: dP (two layouts), dX ----
            ok = mbar_wait(smem_u32(&dp_empty), (g & 1) ^ 1);
            for (int i = tb; i < te; ++i) {
                const int64_t t0 = start + 128 * (int64_t)i;
                const bool active = t0 + row < end;
                const int64_t tok = t0 + row;
                float db[C::R];
                float dp[C::M];
                if (active) {
                    load_bf16_row<C::R>(a.dB + tok * C::R, db);
                    const float4 *ps = reinterpret_cast<const float4 *>(a.P + tok * C::M);
#pragma unroll
                    for (int j = 0; j < C::M / 4; ++j) {
                        const float4 v = ps[j];
                        dp[4 * j] = v.x; dp[4 * j + 1] = v.y; dp[4 * j + 2] = v.z; dp[4 * j + 3] = v.w;
                    }
                } else {
#pragma unroll
                    for (int k = 0; k < C::R; ++k) db[k] = 0.0f;
#pragma unroll
                    for (int j = 0; j < C::M; ++j) dp[j] = 0.0f;
                }
#pragma unroll
                for (int jb = 0; jb < C::M; jb += 16) {
                    float acc[16];
                    vecmat16<C::R, C::M>(db, we2t, jb, acc);   // dA = dB . We2^T
#pragma unroll
                    for (int e = 0; e < 16; ++e) dp[jb + e] = active ? acc[e] * dact_fast(a.act, dp[jb + e]) : 0.0f;
                }
                // dP rows = tokens (K-major over m, DSW-byte rows)
                uint8_t *pa = smem + C::OFF_DPA + (i - tb) * C::DPA_TILE;
#pragma unroll
                for (int cc = 0; cc < C::M / 8; ++cc) {
                    uint32_t pk[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        __nv_bfloat162 h = __floats2bfloat162_rn(dp[8 * cc + 2 * e], dp[8 * cc + 2 * e + 1]);
                        pk[e] = *reinterpret_cast<uint32_t *>(&h);
                    }
                    *reinterpret_cast<uint4 *>(pa + swz_offset(row, 16 * cc, C::DSW)) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
                }
                // dP^T rows = m (K-major over the tile's tokens, 128B rows, two 64-token blocks)
                uint8_t *pt = smem + C::OFF_DPT + (i - tb) * C::DPT_TILE + (row >> 6) * (C::M * 128);
                const uint32_t byte = (row & 63) * 2;
#pragma unroll
                for (int j = 0; j < C::M; ++j)
                    *reinterpret_cast<__nv_bfloat16 *>(pt + swz_offset(j, byte, 128)) = __float2bfloat16_rn(dp[j]);
                // publish this tile's dP so its products can start
                fence_async_smem();
                named_barrier(1, 128);
                if (et == 0) mbar_arrive(smem_u32(&dp_full[i - tb]));
                // identity path: dX[:, :r] += dB
                if (active && a.dX) {
                    uint4 *xp = reinterpret_cast<uint4 *>(a.dX + tok * a.d);
#pragma unroll
                    for (int v = 0; v < C::R / 8; ++v) {
                        float xv[8];
                        load_bf16_row<8>(a.dX + tok * a.d + 8 * v, xv);
                        uint32_t pk[4];
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            __nv_bfloat162 h = __floats2bfloat162_rn(xv[2 * e] + db[8 * v + 2 * e],
                                                                     xv[2 * e + 1] + db[8 * v + 2 * e + 1]);
                            pk[e] = *reinterpret_cast<uint32_t *>(&h);
                        }
                        xp[v] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
                    }
                }
            }

            // ---- phase 1: dF tiles out by TMA; dWe1 chunks to the partial slot ----
            for (int c = 0; c < nch && ok; ++c, ++cit) {
                for (int i = tb; i < te && ok; ++i, ++dfit) {
                    const int64_t t0 = start + 128 * (int64_t)i;
                    const int valid = (int)((end - t0) < 128 ? (end - t0) : 128);
                    const uint32_t ad_buf = dfit & 1;
                    ok = mbar_wait(smem_u32(&df_full[ad_buf]), (dfit >> 1) & 1);
                    tc_fence_after();
#pragma unroll
                    for (int h = 0; h < 2; ++h, ++sit) {
                        const uint32_t sb = sit & 1;
                        if (et == 0) bulk_wait_read<1>();   // staging half sb is free again
                        named_barrier(1, 128);
                        uint8_t *stg = smem + C::OFF_STG + sb * C::STG_HALF;
                        // a warp whose rows all lie past the valid tokens has nothing to store
                        const int gqend = (q * 32 < valid) ? 2 : 0;
#pragma unroll
                        for (int gq = 0; gq < 2; ++gq) {
                            if (gq >= gqend) break;
                            float v[32];
                            tmem_ld32(tmem_df + ((uint32_t)(q * 32) << 16) + ad_buf * 128 + h * 64 + gq * 32, v);
                            tmem_ld_wait();
                            uint32_t p[16];
#pragma unroll
                            for (int e = 0; e < 16; ++e) {
                                __nv_bfloat162 hh = __floats2bfloat162_rn(v[2 * e], v[2 * e + 1]);
                                p[e] = *reinterpret_cast<uint32_t *>(&hh);
                            }
#pragma unroll
                            for (int e = 0; e < 4; ++e)
                                *reinterpret_cast<uint4 *>(stg + swz_offset(row, gq * 64 + 16 * e, 128)) =
                                    make_uint4(p[4 * e], p[4 * e + 1], p[4 * e + 2], p[4 * e + 3]);
                        }
                        if (h == 1) {
                            tc_fence_before();
                            mbar_arrive(smem_u32(&df_empty[ad_buf]));
                        }
                        fence_async_smem();
                        named_barrier(1, 128);
                        if (et == 0) {
                            const int x = c * 128 + 64 * h;
                            if (valid == 128) {
                                tma_store_2d(&tm_df128, x, (int32_t)t0, smem_u32(stg));
                            } else {
                                for (int rg = 0; rg * 16 < valid; ++rg)
                                    tma_store_2d(&tm_df16, x, (int32_t)(t0 + 16 * rg), smem_u32(stg) + rg * 2048);
                            }
                            bulk_commit();
                        }
                    }
                }
                // the chunk's dWe1 rows (lane = d column) -> cross-CTA reduction
                const uint32_t ae = cit & 1;
                ok = ok && mbar_wait(smem_u32(&we_full[ae]), (cit >> 1) & 1);
                tc_fence_after();
                float v[C::M];
#pragma unroll
                for (int j = 0; j < C::M; j += 16) {
                    float t16[16];
                    tmem_ld16(tmem_we + ((uint32_t)(q * 32) << 16) + ae * C::MS + j, t16);
                    tmem_ld_wait();
#pragma unroll
                    for (int e = 0; e < 16; ++e) v[j + e] = t16[e];
                }
                tc_fence_before();
                mbar_arrive(smem_u32(&we_empty[ae]));   // the accumulator is free again
                wgrad_chunk<C::M>(a.wg, v, c, row, g == 0);
            }

            // ---- phase 3: dWe2 partial = sum over tokens of phi(P)^T dB ----
            if (et == 0) bulk_wait_read<0>();   // staging no longer read by TMA stores
            named_barrier(1, 128);
            float *sA = reinterpret_cast<float *>(smem + C::OFF_F);   // [128][M + 1]
            float *sD = sA + 128 * (C::M + 1);                          // [128][R + 1]
            float acc2[NOUT];
#pragma unroll
            for (int k = 0; k < NOUT; ++k) acc2[k] = 0.0f;
            for (int i = tb; i < te; ++i) {
                const int64_t t0 = start + 128 * (int64_t)i;
                const int valid = (int)((end - t0) < 128 ? (end - t0) : 128);
                const bool active = row < valid;
                const int64_t tok = t0 + row;
                float av[C::M], db[C::R];
                if (active) {
                    const float4 *ps = reinterpret_cast<const float4 *>(a.P + tok * C::M);
#pragma unroll
                    for (int j = 0; j < C::M / 4; ++j) {
                        const float4 v = ps[j];
                        av[4 * j] = act_fast(a.act, v.x); av[4 * j + 1] = act_fast(a.act, v.y);
                        av[4 * j + 2] = act_fast(a.act, v.z); av[4 * j + 3] = act_fast(a.act, v.w);
                    }
                    load_bf16_row<C::R>(a.dB + tok * C::R, db);
                } else {
#pragma unroll
                    for (int j = 0; j < C::M; ++j) av[j] = 0.0f;
#pragma unroll
                    for (int k = 0; k < C::R; ++k) db[k] = 0.0f;
                }
                named_barrier(1, 128);
#pragma unroll
                for (int j = 0; j < C::M; ++j) sA[row * (C::M + 1) + j] = av[j];
#pragma unroll
                for (int k = 0; k < C::R; ++k) sD[row * (C::R + 1) + k] = db[k];
                named_barrier(1, 128);
                // output o = et + 128 kk is (j, k) = (o / R, o % R); 128 is a multiple of R, so k
                // is the same for all of this thread's outputs. Each output sums over t in order;
                // the outputs' chains interleave so their latencies overlap.
                {
                    static_assert((C::M * C::R) % 128 == 0 && 128 % C::R == 0, "dWe2 output split");
                    const int k = et % C::R, j0 = et / C::R;
#pragma unroll 2
                    for (int t = 0; t < valid; ++t) {
                        const float dv = sD[t * (C::R + 1) + k];
                        const float *at = sA + t * (C::M + 1) + j0;
#pragma unroll
                        for (int kk = 0; kk < NOUT; ++kk) acc2[kk] = fmaf(at[kk * (128 / C::R)], dv, acc2[kk]);
                    }
                }
            }
#pragma unroll
            for (int kk = 0; kk < NOUT; ++kk) a.part2[slot * (C::M * C::R) + et + 128 * kk] = acc2[kk];
            named_barrier(1, 128);
            if (et == 0) mbar_arrive(smem_u32(&p3_done));
        }
        for (int g = ngroups; g < a.max_groups; ++g) {
            const int64_t slot = (int64_t)blockIdx.x * a.max_groups + g;
            for (int e = et; e < C::M * C::R; e += 128) a.part2[slot * (C::M * C::R) + e] = 0.0f;
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
