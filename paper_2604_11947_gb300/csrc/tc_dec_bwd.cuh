// tc_dec_bwd.cuh -- backward of the receive side on tensor cores (chain rule of Sec. 3.2's
// decoder with the zero-padding identity path of Eq. Pid):
//   G = phi(Q), Q = B . Wd1;  dG = dY . Wd2^T;  dQ = dG * phi'(Q);
//   dB = [merge] dY[:, :r] + dQ . Wd1^T;  dWd2 = G^T . dY;  dWd1 = B^T . dQ.
//
// Persistent CTAs over contiguous 16-token-aligned token ranges, processed in groups of up to
// NT tiles of 128 tokens. For each group:
//   phase 0 (epilogue warps): Q, G on CUDA cores; G^T (m rows x 128 tokens per tile, K-major
//            over tokens, 128B swizzle) into shared memory.
//   phase 1 (producer + MMA): d in chunks of 128 columns; per chunk one Wd2 slice (K-major) and,
//            per tile, one dY tile (128 tokens x 128 columns) feeding two MMAs:
//              dG_tile   (128 tokens x m, TMEM, kept over all chunks) += dY . Wd2_chunk^T
//              dWd2T_chk (128 columns x m, TMEM, double-buffered)     += dY^T . G_tile
//            (the second MMA reads the same shared-memory tile as an MN-major operand).
//            The epilogue warps drain each finished dWd2T chunk to the fp32 partial slot.
//   phase 2 (epilogue warps): dQ, dB, and the dWd1 partial (B^T . dQ summed over the group's
//            tokens in a fixed order, via the then idle dY ring as scratch).
// A second kernel sums the partial slots in a fixed order (deterministic).
// HBM traffic per token: read dY (2d), B (2r), dY[:, :r] again (2r, L2), write dB (2r);
// per slot: d x m + r x m fp32 partials.
#pragma once

#include "common.cuh"
#include "tc_common.cuh"
#include "tc_wgrad.cuh"

namespace resbm {
namespace tc {

template <int M_> struct DecBwdCfg {
    static constexpr int M = M_;
    static constexpr int R = M_;
    static constexpr int MS = M_ < 32 ? 32 : M_;              // TMEM columns per accumulator
    static constexpr int NT = 4;                              // tiles per group
    static constexpr int NSY = M_ <= 32 ? 4 : 3;              // dY ring depth
    static constexpr uint32_t Y_STAGE = 128 * 128 * 2;        // 128 tokens x 128 columns
    static constexpr uint32_t W_STAGE = M_ * 128 * 2;         // m rows x 128 columns
    static constexpr uint32_t GT_TILE = M_ * 128 * 2;         // m rows x 128 tokens
    static constexpr uint32_t WD1_BYTES = R * M_ * 2;
    static constexpr uint32_t OFF_Y = 0;
    static constexpr uint32_t OFF_W = OFF_Y + NSY * Y_STAGE;
    static constexpr int NW = M_ <= 32 ? 4 : 3;               // Wd2 slice ring depth
    static constexpr uint32_t OFF_GT = OFF_W + NW * W_STAGE;
    static constexpr uint32_t OFF_WD1 = OFF_GT + NT * GT_TILE;
    static constexpr uint32_t OFF_WD1T = OFF_WD1 + WD1_BYTES;
    static constexpr uint32_t SMEM_BYTES = OFF_WD1T + WD1_BYTES + 1024;
    static constexpr uint32_t TMEM_NEED = (NT + 2) * MS;
    static constexpr uint32_t TMEM_COLS = TMEM_NEED <= 128 ? 128 : TMEM_NEED <= 256 ? 256 : 512;
    static constexpr uint32_t SCRATCH_BYTES = 128 * (R + M_ + 2) * 4;   // phase 2, inside the dY ring
    static_assert(SCRATCH_BYTES <= NSY * Y_STAGE, "phase-2 scratch must fit in the dY ring");
    static constexpr int THREADS = 192;
};

struct DecBwdArgs {
    const __nv_bfloat16 *B;    // T x r
    const __nv_bfloat16 *Wd1;  // r x m
    const __nv_bfloat16 *dY;   // T x d (first r columns re-read for the identity path)
    __nv_bfloat16 *dB;         // T x r
    WgradArgs wg;              // dWd2^T chunks (d x m), reduced across CTAs
    float *part1;              // slots x r x m   (dWd1 partials)
    int64_t T, d;
    int act, merge, max_groups;
};

template <int M_>
__global__ void __launch_bounds__(192, 1)
    k_dec_bwd(const __grid_constant__ CUtensorMap tm_dy128, const __grid_constant__ CUtensorMap tm_dy16,
              const __grid_constant__ CUtensorMap tm_wd2, const DecBwdArgs a)
{
    using C = DecBwdCfg<M_>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    __shared__ uint64_t y_full[C::NSY], y_empty[C::NSY], w_full[C::NW], w_empty[C::NW];
    __shared__ uint64_t gt_full[C::NT], gt_empty, wt_full[2], wt_empty[2], dg_full, dg_empty, p2_done, done_bar;
    __shared__ uint32_t tmem_base_sh;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nch = (int)(a.d / 128);
    int64_t start, end;
    token_range(a.T, blockIdx.x, gridDim.x, start, end);
    const int ntiles = (int)((end - start + 127) / 128);
    const int ngroups = (ntiles + C::NT - 1) / C::NT;

    if (threadIdx.x == 0) {
        for (int s = 0; s < C::NSY; ++s) {
            mbar_init(smem_u32(&y_full[s]), 1);
            mbar_init(smem_u32(&y_empty[s]), 1);
        }
        for (int i = 0; i < C::NW; ++i) {
            mbar_init(smem_u32(&w_full[i]), 1);
            mbar_init(smem_u32(&w_empty[i]), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(smem_u32(&wt_full[i]), 1);
            mbar_init(smem_u32(&wt_empty[i]), 128);
        }
        for (int i = 0; i < C::NT; ++i) mbar_init(smem_u32(&gt_full[i]), 1);
        mbar_init(smem_u32(&gt_empty), 1);
        mbar_init(smem_u32(&dg_full), 1);
        mbar_init(smem_u32(&dg_empty), 128);
        mbar_init(smem_u32(&p2_done), 1);
        mbar_init(smem_u32(&done_bar), 1);
        fence_mbar_init();
    }
    if (warp == 1) tmem_alloc(smem_u32(&tmem_base_sh), C::TMEM_COLS);
    if (warp >= 2) {  // Wd1 (r x m) and its transpose (m x r), bf16, into shared memory
        const uint4 *src = reinterpret_cast<const uint4 *>(a.Wd1);
        uint4 *dst = reinterpret_cast<uint4 *>(smem + C::OFF_WD1);
        for (int i = threadIdx.x - 64; i < (int)(C::WD1_BYTES / 16); i += 128) dst[i] = src[i];
        __nv_bfloat16 *dt = reinterpret_cast<__nv_bfloat16 *>(smem + C::OFF_WD1T);
        for (int e = threadIdx.x - 64; e < C::R * C::M; e += 128) dt[(e % C::M) * C::R + e / C::M] = a.Wd1[e];
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_base_sh;
    const uint32_t tmem_dg = tmem;                     // NT accumulators of MS columns
    const uint32_t tmem_wt = tmem + C::NT * C::MS;     // 2 accumulators of MS columns

    if (warp == 0) {
        // ---------------- producer ----------------
        if (elect_one()) {
            tma_prefetch_desc(&tm_dy128);
            tma_prefetch_desc(&tm_dy16);
            tma_prefetch_desc(&tm_wd2);
            uint32_t yit = 0, wit = 0;
            bool ok = true;
            for (int g = 0; g < ngroups && ok; ++g) {
                if (g > 0) ok = mbar_wait(smem_u32(&p2_done), (g - 1) & 1);  // the ring was scratch
                const int tb = g * C::NT, te = min(ntiles, tb + C::NT);
                for (int c = 0; c < nch && ok; ++c) {
                    // order: dY tile 0 of the chunk, the chunk's Wd2 slice, the other dY tiles.
                    // The MMA needs the slice before any tile of the chunk, so it must not queue
                    // behind tiles that wait for ring slots (that would deadlock), and it must not
                    // delay the first tile (that would stall the stream on the small weight ring).
                    for (int i = tb; i < te; ++i) {
                        if (i == tb + 1) {
                            const uint32_t s = wit % C::NW, ph = (wit / C::NW) & 1;
                            if (!mbar_wait(smem_u32(&w_empty[s]), ph ^ 1)) { ok = false; break; }
                            const uint32_t dst = smem_u32(smem + C::OFF_W + s * C::W_STAGE);
                            mbar_expect_tx(smem_u32(&w_full[s]), C::W_STAGE);
                            for (int h = 0; h < 2; ++h)
                                tma_load_2d(dst + h * (C::M * 128), &tm_wd2, c * 128 + 64 * h, 0, smem_u32(&w_full[s]));
                            ++wit;
                        }
                        const int64_t t0 = start + 128 * (int64_t)i;
                        const int valid = (int)((end - t0) < 128 ? (end - t0) : 128);
                        const int nb = (valid + 15) / 16;
                        const uint32_t s = yit % C::NSY, ph = (yit / C::NSY) & 1;
                        if (!mbar_wait(smem_u32(&y_empty[s]), ph ^ 1)) { ok = false; break; }
                        const uint32_t dst = smem_u32(smem + C::OFF_Y + s * C::Y_STAGE);
                        const uint32_t bar = smem_u32(&y_full[s]);
                        mbar_expect_tx(bar, valid == 128 ? C::Y_STAGE : (uint32_t)nb * 2u * 2048u);
                        for (int h = 0; h < 2; ++h) {
                            if (valid == 128) {
                                tma_load_2d(dst + h * 16384, &tm_dy128, c * 128 + 64 * h, (int32_t)t0, bar);
                            } else {
                                for (int rg = 0; rg < nb; ++rg)
                                    tma_load_2d(dst + h * 16384 + rg * 2048, &tm_dy16, c * 128 + 64 * h,
                                                (int32_t)(t0 + 16 * rg), bar);
                            }
                        }
                        ++yit;
                    }
                    if (!ok) break;
                    if (te - tb == 1) {  // a one-tile group: the slice after its only tile
                        const uint32_t s = wit % C::NW, ph = (wit / C::NW) & 1;
                        if (!mbar_wait(smem_u32(&w_empty[s]), ph ^ 1)) { ok = false; break; }
                        const uint32_t dst = smem_u32(smem + C::OFF_W + s * C::W_STAGE);
                        mbar_expect_tx(smem_u32(&w_full[s]), C::W_STAGE);
                        for (int h = 0; h < 2; ++h)
                            tma_load_2d(dst + h * (C::M * 128), &tm_wd2, c * 128 + 64 * h, 0, smem_u32(&w_full[s]));
                        ++wit;
                    }
                }
            }
            // drain the loads still in flight
            for (uint32_t k = 0; k < (yit < (uint32_t)C::NSY ? yit : (uint32_t)C::NSY); ++k) {
                const uint32_t j = yit - 1 - k;
                mbar_wait(smem_u32(&y_full[j % C::NSY]), (j / C::NSY) & 1);
            }
            for (uint32_t k = 0; k < (wit < (uint32_t)C::NW ? wit : (uint32_t)C::NW); ++k) {
                const uint32_t j = wit - 1 - k;
                mbar_wait(smem_u32(&w_full[j % C::NW]), (j / C::NW) & 1);
            }
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if (elect_one()) {
            constexpr uint32_t id_dg = idesc_bf16(128, C::M, false, false);  // dY (K-major) . Wd2 (K-major)
            constexpr uint32_t id_wt = idesc_bf16(128, C::M, true, false);   // dY^T (MN-major) . G^T (K-major)
            // shared-memory descriptors of ring slot 0, advanced per slot and K step by adding the
            // byte offset >> 4 to the start-address field (no carry: shared addresses < 256 KB)
            const uint64_t yk0 = smem_desc(smem_u32(smem + C::OFF_Y), 16, 1024, kSwz128);     // dY, K-major
            const uint64_t ym0 = smem_desc(smem_u32(smem + C::OFF_Y), 16384, 1024, kSwz128);  // dY, MN-major
            const uint64_t wk0 = smem_desc(smem_u32(smem + C::OFF_W), 16, 1024, kSwz128);     // Wd2 slice
            const uint64_t gk0 = smem_desc(smem_u32(smem + C::OFF_GT), 16, 1024, kSwz128);    // G^T tiles
            uint32_t yit = 0, wit = 0, cit = 0;
            bool ok = true;
            for (int g = 0; g < ngroups && ok; ++g) {
                const int tb = g * C::NT, te = min(ntiles, tb + C::NT);
                if (g > 0) ok = mbar_wait(smem_u32(&dg_empty), (g - 1) & 1);
                tc_fence_after();
                for (int c = 0; c < nch && ok; ++c, ++cit) {
                    const uint32_t sw = wit % C::NW;
                    const uint32_t ab = cit & 1;
                    ok = mbar_wait(smem_u32(&w_full[sw]), (wit / C::NW) & 1) &&
                         mbar_wait(smem_u32(&wt_empty[ab]), ((cit >> 1) & 1) ^ 1);
                    tc_fence_after();
                    const uint64_t wk = wk0 + ((sw * C::W_STAGE) >> 4);
                    const uint32_t d_wt = tmem_wt + ab * C::MS;
                    for (int i = tb; i < te && ok; ++i, ++yit) {
                        const int64_t t0 = start + 128 * (int64_t)i;
                        const int valid = (int)((end - t0) < 128 ? (end - t0) : 128);
                        const uint32_t s = yit % C::NSY;
                        ok = mbar_wait(smem_u32(&y_full[s]), (yit / C::NSY) & 1);
                        tc_fence_after();
                        const uint64_t yk = yk0 + ((s * C::Y_STAGE) >> 4);
                        const uint64_t ym = ym0 + ((s * C::Y_STAGE) >> 4);
                        const uint64_t gk = gk0 + (((i - tb) * C::GT_TILE) >> 4);
                        const uint32_t d_dg = tmem_dg + (i - tb) * C::MS;
                        // dG_tile += dY_tile . Wd2_chunk^T: K = 128 columns in 8 steps of 16
                        mma_bf16(d_dg, yk, wk, id_dg, c != 0);
#pragma unroll
                        for (int k = 1; k < 8; ++k)
                            mma_bf16(d_dg, yk + kmaj_off(k, 16384), wk + kmaj_off(k, C::M * 128), id_dg, true);
                        // the dWd2 product needs the tile's G^T (published per tile in phase 0,
                        // once per group; the dG products above did not wait for it)
                        if (c == 0) {
                            ok = ok && mbar_wait(smem_u32(&gt_full[i - tb]), g & 1);
                            tc_fence_after();
                        }
                        // dWd2T_chunk += dY_tile^T . G_tile: K = the tile's tokens in steps of 16
                        if (valid == 128) {
#pragma unroll
                            for (int k = 0; k < 8; ++k)
                                mma_bf16(d_wt, ym + ((k * 2048) >> 4), gk + kmaj_off(k, C::M * 128), id_wt,
                                         (i > tb) || (k > 0));
                        } else {
                            const int nks = (valid + 15) / 16;
                            for (int k = 0; k < nks; ++k)
                                mma_bf16(d_wt, ym + ((k * 2048) >> 4), gk + kmaj_off(k, C::M * 128), id_wt,
                                         (i > tb) || (k > 0));
                        }
                        mma_commit(smem_u32(&y_empty[s]));
                    }
                    mma_commit(smem_u32(&w_empty[sw]));
                    mma_commit(smem_u32(&wt_full[ab]));
                    ++wit;
                }
                mma_commit(smem_u32(&gt_empty));
                mma_commit(smem_u32(&dg_full));
            }
            mma_commit(smem_u32(&done_bar));
            mbar_wait(smem_u32(&done_bar), 0);
        }
    } else {
        // ---------------- epilogue warps ----------------
        const int q = warp & 3;
        const int row = q * 32 + lane;  // token row (phases 0, 2) or d-column row (phase 1)
        const int et = threadIdx.x - 64;
        const __nv_bfloat16 *wd1 = reinterpret_cast<const __nv_bfloat16 *>(smem + C::OFF_WD1);    // r x m
        const __nv_bfloat16 *wd1t = reinterpret_cast<const __nv_bfloat16 *>(smem + C::OFF_WD1T);  // m x r
        constexpr int NOUT = (C::R * C::M + 127) / 128;  // dWd1 outputs per thread
        uint32_t cit = 0;
        bool ok = true;
        for (int g = 0; g < ngroups && ok; ++g) {
            const int tb = g * C::NT, te = min(ntiles, tb + C::NT);
            const int64_t slot = (int64_t)blockIdx.x * a.max_groups + g;
            // ---- phase 0: G^T of every tile of the group ----
            ok = mbar_wait(smem_u32(&gt_empty), (g & 1) ^ 1);
            for (int i = tb; i < te; ++i) {
                const int64_t t0 = start + 128 * (int64_t)i;
                const bool active = t0 + row < end;
                float bq[C::R];
                if (active) {
                    load_bf16_row<C::R>(a.B + (t0 + row) * C::R, bq);
                } else {
#pragma unroll
                    for (int k = 0; k < C::R; ++k) bq[k] = 0.0f;
                }
                uint8_t *gt = smem + C::OFF_GT + (i - tb) * C::GT_TILE + (row >> 6) * (C::M * 128);
                const uint32_t byte = (row & 63) * 2;
#pragma unroll
                for (int jb = 0; jb < C::M; jb += 16) {
                    float acc[16];
                    vecmat16<C::R, C::M>(bq, wd1, jb, acc);   // Q = B . Wd1
#pragma unroll
                    for (int e = 0; e < 16; ++e) {
                        const float gv = active ? act_fast(a.act, acc[e]) : 0.0f;
                        *reinterpret_cast<__nv_bfloat16 *>(gt + swz_offset(jb + e, byte, 128)) = __float2bfloat16_rn(gv);
                    }
                }
                // publish this tile's G^T so its first dWd2 product can start
                fence_async_smem();
                named_barrier(1, 128);
                if (et == 0) mbar_arrive(smem_u32(&gt_full[i - tb]));
            }

            // ---- phase 1: drain each chunk's dWd2^T partial ----
            for (int c = 0; c < nch && ok; ++c, ++cit) {
                const uint32_t ab = cit & 1;
                ok = mbar_wait(smem_u32(&wt_full[ab]), (cit >> 1) & 1);
                tc_fence_after();
                float v[C::M];
#pragma unroll
                for (int j = 0; j < C::M; j += 16) {
                    float t16[16];
                    tmem_ld16(tmem_wt + ((uint32_t)(q * 32) << 16) + ab * C::MS + j, t16);
                    tmem_ld_wait();
#pragma unroll
                    for (int e = 0; e < 16; ++e) v[j + e] = t16[e];
                }
                tc_fence_before();
                mbar_arrive(smem_u32(&wt_empty[ab]));   // the accumulator is free again
                wgrad_chunk<C::M>(a.wg, v, c, row, g == 0);
            }

            // ---- phase 2: dQ, dB, dWd1 partial ----
            ok = ok && mbar_wait(smem_u32(&dg_full), g & 1);
            tc_fence_after();
            // scratch rows padded by one float so that a warp's row-wise stores hit distinct banks
            float *sB = reinterpret_cast<float *>(smem + C::OFF_Y);   // [128][R + 1]
            float *sQ = sB + 128 * (C::R + 1);                          // [128][M + 1]
            float acc1[NOUT];
#pragma unroll
            for (int k = 0; k < NOUT; ++k) acc1[k] = 0.0f;
            for (int i = tb; i < te; ++i) {
                const int64_t t0 = start + 128 * (int64_t)i;
                const int valid = (int)((end - t0) < 128 ? (end - t0) : 128);
                const bool active = row < valid;
                const int64_t tok = t0 + row;
                float dq[C::M];
#pragma unroll
                for (int j = 0; j < C::M; j += 16) {
                    float t16[16];
                    tmem_ld16(tmem_dg + ((uint32_t)(q * 32) << 16) + (i - tb) * C::MS + j, t16);
                    tmem_ld_wait();
#pragma unroll
                    for (int e = 0; e < 16; ++e) dq[j + e] = t16[e];
                }
                float bq[C::R];
                if (active) {
                    load_bf16_row<C::R>(a.B + tok * C::R, bq);
                } else {
#pragma unroll
                    for (int k = 0; k < C::R; ++k) bq[k] = 0.0f;
                }
                // dQ = dG * phi'(Q), Q recomputed from B
#pragma unroll
                for (int jb = 0; jb < C::M; jb += 16) {
                    float acc[16];
                    vecmat16<C::R, C::M>(bq, wd1, jb, acc);
#pragma unroll
                    for (int e = 0; e < 16; ++e) dq[jb + e] = active ? dq[jb + e] * dact_fast(a.act, acc[e]) : 0.0f;
                }
                if (active) {
                    // dB = [merge] dY[:, :r] + dQ . Wd1^T
                    uint4 *dbo = reinterpret_cast<uint4 *>(a.dB + tok * C::R);
#pragma unroll
                    for (int ib = 0; ib < C::R; ib += 16) {
                        float o[16];
                        vecmat16<C::M, C::R>(dq, wd1t, ib, o);
                        if (a.merge) {
                            float y[16];
                            load_bf16_row<16>(a.dY + tok * a.d + ib, y);
#pragma unroll
                            for (int e = 0; e < 16; ++e) o[e] = y[e] + o[e];
                        }
                        uint32_t pk[8];
#pragma unroll
                        for (int e = 0; e < 8; ++e) {
                            __nv_bfloat162 hh = __floats2bfloat162_rn(o[2 * e], o[2 * e + 1]);
                            pk[e] = *reinterpret_cast<uint32_t *>(&hh);
                        }
                        dbo[ib / 8] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
                        dbo[ib / 8 + 1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
                    }
                }
                // dWd1 partial: sum over the tile's tokens of B[t][k] dQ[t][j], in token order
                named_barrier(1, 128);   // the previous tile's scratch reads are done
#pragma unroll
                for (int k = 0; k < C::R; ++k) sB[row * (C::R + 1) + k] = bq[k];
#pragma unroll
                for (int j = 0; j < C::M; ++j) sQ[row * (C::M + 1) + j] = dq[j];
                named_barrier(1, 128);
                // output o = et + 128 kk is (ki, j) = (o / M, o % M); 128 is a multiple of M, so j
                // is the same for all of this thread's outputs. Each output sums over t in order;
                // the outputs' chains interleave so their latencies overlap.
                {
                    static_assert((C::R * C::M) % 128 == 0 && 128 % C::M == 0, "dWd1 output split");
                    const int j = et % C::M, ki0 = et / C::M;
#pragma unroll 2
                    for (int t = 0; t < valid; ++t) {
                        const float qv = sQ[t * (C::M + 1) + j];
                        const float *bt = sB + t * (C::R + 1) + ki0;
#pragma unroll
                        for (int kk = 0; kk < NOUT; ++kk) acc1[kk] = fmaf(bt[kk * (128 / C::M)], qv, acc1[kk]);
                    }
                }
            }
            tc_fence_before();
            mbar_arrive(smem_u32(&dg_empty));
#pragma unroll
            for (int kk = 0; kk < NOUT; ++kk) a.part1[slot * (C::R * C::M) + et + 128 * kk] = acc1[kk];
            named_barrier(1, 128);   // scratch reads done before the ring is reused
            if (et == 0) mbar_arrive(smem_u32(&p2_done));
        }
        // slots of groups this CTA does not have: zeros
        for (int g = ngroups; g < a.max_groups; ++g) {
            const int64_t slot = (int64_t)blockIdx.x * a.max_groups + g;
            for (int e = et; e < C::R * C::M; e += 128) a.part1[slot * (C::R * C::M) + e] = 0.0f;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, C::TMEM_COLS);
    }
}

// out = sum over slots s = 0, 1, ... of part[s] (rows x cols each, rows * cols % 4 == 0), each
// element summed in slot order. Four consecutive elements per thread (16-byte loads) and eight
// slots loaded ahead keep enough reads in flight. With transpose the result is written
// cols x rows (part slices are d x m, the weight gradient is m x d); out4 says out is 16-byte
// aligned (untransposed only).
__device__ __forceinline__ void add4(float4 &a, const float4 &b)
{
    a.x += b.x; a.y += b.y; a.z += b.z; a.w += b.w;
}

// Fixed-order sum of `slots` partial fp32 matrices (rows x cols, cols % 4 == 0) into `out`
// (transposed to cols x rows if `transpose`; `out4`: out is 16-byte aligned). A block of
// 32 x kSlotGroups threads owns 32 consecutive float4 columns of the flattened matrix; thread
// row g sums the g-th contiguous range of slots in slot order, and the groups' sums are then
// added in group order: the same order for every launch, so results are bitwise reproducible.
constexpr int kSlotGroups = 16;

__global__ void __launch_bounds__(32 * kSlotGroups) k_reduce_slots(const float *__restrict__ part, int64_t slots,
                                                                   int64_t rows, int64_t cols,
                                                                   float *__restrict__ out, int transpose, int out4)
{
    __shared__ float4 grp[kSlotGroups][32];
    const int64_t n4 = rows * cols / 4;
    const float4 *p4 = reinterpret_cast<const float4 *>(part);
    const int64_t per = (slots + kSlotGroups - 1) / kSlotGroups;
    const int64_t s0 = threadIdx.y * per;
    const int64_t s1 = s0 + per < slots ? s0 + per : slots;
    for (int64_t base = (int64_t)blockIdx.x * 32; base < n4; base += (int64_t)gridDim.x * 32) {
        const int64_t e4 = base + threadIdx.x;
        float4 acc = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
        if (e4 < n4) {
            int64_t s = s0;
            for (; s + 4 <= s1; s += 4) {
                float4 v[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) v[u] = __ldcs(&p4[(s + u) * n4 + e4]);
#pragma unroll
                for (int u = 0; u < 4; ++u) add4(acc, v[u]);
            }
            for (; s < s1; ++s) add4(acc, __ldcs(&p4[s * n4 + e4]));
        }
        grp[threadIdx.y][threadIdx.x] = acc;
        __syncthreads();
        if (threadIdx.y == 0 && e4 < n4) {
            float4 t = grp[0][threadIdx.x];
#pragma unroll
            for (int g = 1; g < kSlotGroups; ++g) add4(t, grp[g][threadIdx.x]);
            const int64_t e = 4 * e4;
            if (transpose) {
                const int64_t rr = e / cols, cc = e - rr * cols;
                out[(cc + 0) * rows + rr] = t.x;
                out[(cc + 1) * rows + rr] = t.y;
                out[(cc + 2) * rows + rr] = t.z;
                out[(cc + 3) * rows + rr] = t.w;
            } else if (out4) {
                reinterpret_cast<float4 *>(out)[e4] = t;
            } else {
                out[e] = t.x; out[e + 1] = t.y; out[e + 2] = t.z; out[e + 3] = t.w;
            }
        }
        __syncthreads();
    }
}

}  // namespace tc
}  // namespace resbm
