// tc_dec_bwd.cuh -- backward of the receive side on tensor cores (chain rule of Sec. 3.2's
// decoder with the zero-padding identity path of Eq. Pid):
//   Q = B . Wd1, G = phi(Q);  dG = dY . Wd2^T;  dQ = dG * phi'(Q);
//   dB = [merge] dY[:, :r] + dQ . Wd1^T;  dWd2 = G^T . dY;  dWd1 = B^T . dQ.
//
// Persistent CTAs (in clusters of 1, 2 or 4) over contiguous runs of whole 128-token tiles,
// processed in groups of up to NT tiles of 128 tokens (every CTA has the same number of groups,
// its tiles split evenly). Every product runs on tcgen05; the CUDA cores only apply phi and phi'
// and convert. For each group:
//   phase 0: the group's B tiles (TMA) -> Q_tile = B . Wd1 in TMEM (kept for phase 2) -> the
//            epilogue writes G = phi(Q) as a bf16 pair hi + lo, rows [token][m], to shared
//            memory (hi in the G tiles, lo over the B tiles, which the Q products have read).
//   phase 1: d in chunks of 128 columns; per chunk one Wd2 slice and, per tile, one dY tile
//            (128 tokens x 128 columns) feeding the MMAs:
//              dG_tile   (128 tokens x m, TMEM, kept over all chunks) += dY . Wd2_chunk^T
//              dWd2T_chk (128 columns x m, TMEM, double-buffered)     += dY^T . (G_hi + G_lo)
//            (the same dY stage read K-major and MN-major; G read MN-major; dWd2 is a sum over
//            all tokens whose terms cancel strongly for real gradients, so G enters it to about
//            16 significant bits). The epilogue
//            drains each finished dWd2T chunk into the cluster's fp32 partial slot (summed over
//            the cluster's CTAs through distributed shared memory, tc_wgrad.cuh).
//   phase 2: the epilogue writes dQ = dG * phi'(Q) as two bf16 tiles hi + lo (rows [token][m],
//            in the idle dY ring; hi = dQ rounded to bf16, lo = the rounded remainder, so the
//            products see dQ to about 16 significant bits: dB crosses the boundary and is
//            rounded again there) -> dB_tile = dQ . Wd1^T (into the tile's dG columns) and
//            dWd1 += B^T . dQ over the group's tokens (the B tile read MN-major as a 128-row
//            operand whose rows >= r are never read back; the B tiles are loaded again for this
//            phase, into a region idle in it) -> the epilogue adds [merge] dY[:, :r] (a TMA
//            tile) and stores dB as bf16; the group's dWd1 goes to its slot.
// A second kernel sums the partial slots in a fixed order (deterministic).
// HBM traffic per token: read dY (2d), B (2r), dY[:, :r] again (2r, mostly L2), write dB (2r);
// per cluster: d x m fp32 partials; per CTA and group: r x m.
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
    static constexpr int NT = M_ <= 32 ? 4 : 2;               // tiles per group
    static constexpr int NSY = M_ <= 32 ? 4 : 3;              // dY ring depth
    static constexpr int NW = M_ <= 16 ? 4 : M_ <= 32 ? 2 : 3;  // Wd2 slice ring depth
    static constexpr int CLMAX = M_ <= 32 ? 4 : 1;            // CTAs per cluster (weight-gradient exchange)
    static constexpr int CL_MIN_TOKENS = 160;                 // clusters only from this many tokens per CTA
    static constexpr int NWB = CLMAX > 1 ? 3 : 2;             // dWd2T accumulators in TMEM
    static constexpr uint32_t RB = M_ * 2;                    // row bytes (= swizzle) of the r / m wide tiles
    static constexpr uint32_t Y_STAGE = 128 * 128 * 2;        // 128 tokens x 128 columns
    static constexpr uint32_t W_STAGE = M_ * 128 * 2;         // m rows x 128 columns
    static constexpr uint32_t TILE = 128 * RB;                // 128 tokens x r (or m) columns
    static constexpr uint32_t WD1_BYTES = R * M_ * 2;
    static constexpr uint32_t OFF_Y = 0;
    static constexpr uint32_t OFF_W = OFF_Y + NSY * Y_STAGE;
    static constexpr uint32_t OFF_G = OFF_W + NW * W_STAGE;   // G tiles [token][m]
    static constexpr uint32_t OFF_B = OFF_G + NT * TILE;      // B tiles [token][r] (TMA)
    static constexpr uint32_t OFF_WD1 = OFF_B + NT * TILE;    // Wd1 [r][m]: K-major B operand of dQ . Wd1^T
    static constexpr uint32_t OFF_WD1T = OFF_WD1 + WD1_BYTES; // Wd1^T [m][r]: K-major B operand of B . Wd1
    static constexpr uint32_t OFF_RX = OFF_WD1T + WD1_BYTES;  // weight-gradient receive buffer
    static constexpr uint32_t SMEM_BYTES = OFF_RX + wgrad_rx_bytes<M_>(CLMAX) + 1024;
    // phase-2 scratch in the idle dY ring: dQ hi tiles (slot 0), dY[:, :r] tiles (slot 1),
    // dQ lo tiles (slot 2)
    static constexpr uint32_t OFF_DQ = OFF_Y;
    static constexpr uint32_t OFF_YR = OFF_Y + Y_STAGE;
    static constexpr uint32_t OFF_DQLO = OFF_Y + 2 * Y_STAGE;
    static_assert(NT * TILE <= Y_STAGE && NSY >= 3, "phase-2 scratch must fit in three ring slots");
    // G_lo tiles (phase 1) over the B tiles; the B tiles of phase 2 in the fourth ring slot, or in
    // the Wd2 slice ring (both idle in phase 2)
    static constexpr uint32_t OFF_GLO = OFF_B;
    static constexpr uint32_t OFF_B2 = NSY >= 4 ? OFF_Y + 3 * Y_STAGE : OFF_W;
    static_assert(NSY >= 4 ? NT * TILE <= Y_STAGE : NT * TILE <= NW * W_STAGE, "phase-2 B tiles");
    static_assert(SMEM_BYTES <= 232448 - 512, "shared memory budget");
    // dWd2^T products against G_hi and G_lo: for m <= 32 as ONE product with the two tiles as
    // the two swizzle blocks of an N = 2m operand (the accumulator's columns [0, m) and [m, 2m)
    // are the hi and lo parts, added by the epilogue), else as two products into one accumulator
    static constexpr bool WIDE = M_ <= 32;
    static constexpr int MSW = WIDE ? (2 * M_ < 32 ? 32 : 2 * M_) : MS;   // TMEM columns per dWd2T accumulator
    // TMEM columns: dG (later dB) NT x MS | Q NT x MS | dWd2T NWB x MSW | dWd1 MS
    static constexpr uint32_t TM_DG = 0, TM_Q = NT * MS, TM_WT = 2 * NT * MS, TM_W1 = TM_WT + NWB * MSW;
    static constexpr uint32_t TMEM_NEED = TM_W1 + MS;
    static_assert(TMEM_NEED <= 512, "TMEM budget");
    static constexpr uint32_t TMEM_COLS = TMEM_NEED <= 128 ? 128 : TMEM_NEED <= 256 ? 256 : 512;
    static constexpr int THREADS = 192;
};

struct DecBwdArgs {
    const __nv_bfloat16 *Wd1;  // r x m
    __nv_bfloat16 *dB;         // T x r
    WgradArgs wg;              // dWd2^T chunks (d x m), reduced across CTAs
    float *part1;              // slots x r x m   (dWd1 partials)
    int64_t T, d;
    int act, merge, max_groups;
    // 1: the previous kernel of the stream neither writes what this one reads nor reads what it
    // writes (the boundary step's decoder forward), and what this one reads was complete when
    // that kernel passed its own wait: start without waiting for it, and wait for it at the end
    int after_independent;
};

template <int M_>
__global__ void __launch_bounds__(192, 1)
    k_dec_bwd(const __grid_constant__ CUtensorMap tm_dy128, const __grid_constant__ CUtensorMap tm_dy16,
              const __grid_constant__ CUtensorMap tm_wd2, const __grid_constant__ CUtensorMap tm_b,
              const __grid_constant__ CUtensorMap tm_yr, const DecBwdArgs a)
{
    using C = DecBwdCfg<M_>;
    if (!a.after_independent) griddep_wait();   // the previous kernel of the stream has completed
    griddep_launch_dependents();  // the next one may be scheduled on SMs as they free up
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    __shared__ uint64_t y_full[C::NSY], y_empty[C::NSY], w_full[C::NW], w_empty[C::NW];
    __shared__ uint64_t b_full, q_full, g_full[C::NT], g_empty, wt_full[C::NWB], wt_empty[C::NWB], dg_full, dg_empty;
    __shared__ uint64_t yr_full, dq_full[C::NT], db_full[C::NT], w1_full, p2_done, done_bar;
    __shared__ uint64_t rx_full, rx_free[4];
    __shared__ uint32_t tmem_base_sh;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nch = (int)(a.d / 128);
    // every CTA walks the d chunks in the same cyclic order but from its own starting chunk,
    // so that at any moment the CTAs read different column ranges of their rows
    // (per cluster: the CTAs of a cluster exchange the same chunk at the same time)
    const int c_first = (int)(cluster_index() % (unsigned)nch);
    int64_t start, end;
    token_range(a.T, blockIdx.x, gridDim.x, start, end);
    const int ntiles = (int)((end - start + 127) / 128);
    // the same number of tile groups in every CTA (1 .. NT tiles each, checked)
    int ngroups = a.max_groups;
    if (ntiles < ngroups || ntiles > C::NT * ngroups) {
        if (threadIdx.x == 0) flag_error(kErrPlan);
        ngroups = 0;
    }
    WgradXchg<C::M, C::CLMAX> xg{C::CLMAX > 1 ? cluster_size() : 1u, cluster_rank(), cluster_index(),
                                 smem_u32(smem + C::OFF_RX), smem_u32(&rx_full), smem_u32(&rx_free[0]), 0};

    if (threadIdx.x == 0) {
        for (int s = 0; s < C::NSY; ++s) {
            mbar_init(smem_u32(&y_full[s]), 1);
            mbar_init(smem_u32(&y_empty[s]), 1);
        }
        for (int i = 0; i < C::NW; ++i) {
            mbar_init(smem_u32(&w_full[i]), 1);
            mbar_init(smem_u32(&w_empty[i]), 1);
        }
        for (int i = 0; i < C::NWB; ++i) {
            mbar_init(smem_u32(&wt_full[i]), 1);
            mbar_init(smem_u32(&wt_empty[i]), 128);
        }
        for (int i = 0; i < C::NT; ++i) {
            mbar_init(smem_u32(&g_full[i]), 1);
            mbar_init(smem_u32(&dq_full[i]), 1);
            mbar_init(smem_u32(&db_full[i]), 1);
        }
        mbar_init(smem_u32(&b_full), 1);
        mbar_init(smem_u32(&q_full), 1);
        mbar_init(smem_u32(&g_empty), 1);
        mbar_init(smem_u32(&dg_full), 1);
        mbar_init(smem_u32(&dg_empty), 128);
        mbar_init(smem_u32(&yr_full), 1);
        mbar_init(smem_u32(&w1_full), 1);
        mbar_init(smem_u32(&p2_done), 1);
        mbar_init(smem_u32(&done_bar), 1);
        xg.init_barriers();
        fence_mbar_init();
        xg.arm_first();
    }
    if (warp == 1) tmem_alloc(smem_u32(&tmem_base_sh), C::TMEM_COLS);
    if (warp >= 2) {  // Wd1 (r x m) and Wd1^T (m x r) as swizzled K-major operands
        const int et = threadIdx.x - 64;
        for (int e = et; e < C::R * C::M; e += 128) {
            const int i = e / C::M, j = e % C::M;
            const __nv_bfloat16 v = a.Wd1[e];
            *reinterpret_cast<__nv_bfloat16 *>(smem + C::OFF_WD1 + swz_offset(i, 2 * j, C::RB)) = v;
            *reinterpret_cast<__nv_bfloat16 *>(smem + C::OFF_WD1T + swz_offset(j, 2 * i, C::RB)) = v;
        }
        fence_async_smem();
    }
    tc_fence_before();
    __syncthreads();
    if (C::CLMAX > 1 && xg.cl > 1) cluster_sync();   // every CTA's barriers are initialized before any exchange
    tc_fence_after();
    const uint32_t tmem = tmem_base_sh;

    if (warp == 0) {
        // ---------------- producer ----------------
        if (elect_one()) {
            const uint64_t stream_pol = l2_evict_first();   // read once
            tma_prefetch_desc(&tm_dy128);
            tma_prefetch_desc(&tm_dy16);
            tma_prefetch_desc(&tm_wd2);
            tma_prefetch_desc(&tm_b);
            tma_prefetch_desc(&tm_yr);
            uint32_t yit = 0, wit = 0;
            int b_issued = 0, yr_issued = 0;
            bool ok = true;
            for (int g = 0; g < ngroups && ok; ++g) {
                // the ring, the B tiles and the phase-2 scratch of the previous group are free
                if (g > 0) ok = mbar_wait(smem_u32(&p2_done), (g - 1) & 1);
                if (!ok) break;
                int tb, te;
                group_tiles(g, ngroups, ntiles, tb, te);
                // the group's B tiles (128-row boxes: rows past T read as zeros, rows past this
                // CTA's range are loaded but never used)
                mbar_expect_tx(smem_u32(&b_full), (uint32_t)(te - tb) * C::TILE);
                for (int i = tb; i < te; ++i)
                    tma_load_2d(smem_u32(smem + C::OFF_B + (i - tb) * C::TILE), &tm_b, 0,
                                (int32_t)(start + 128 * (int64_t)i), smem_u32(&b_full));
                ++b_issued;
                for (int c = 0; c < nch && ok; ++c) {
                    const int cc = c + c_first < nch ? c + c_first : c + c_first - nch;
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
                                tma_load_2d(dst + h * (C::M * 128), &tm_wd2, cc * 128 + 64 * h, 0, smem_u32(&w_full[s]));
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
                                tma_load_2d_hint(dst + h * 16384, &tm_dy128, cc * 128 + 64 * h, (int32_t)t0, bar, stream_pol);
                            } else {
                                for (int rg = 0; rg < nb; ++rg)
                                    tma_load_2d_hint(dst + h * 16384 + rg * 2048, &tm_dy16, cc * 128 + 64 * h,
                                                (int32_t)(t0 + 16 * rg), bar, stream_pol);
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
                            tma_load_2d(dst + h * (C::M * 128), &tm_wd2, cc * 128 + 64 * h, 0, smem_u32(&w_full[s]));
                        ++wit;
                    }
                }
                if (!ok) break;
                // dY[:, :r] tiles for phase 2, into ring slot 1 once the group's MMAs are done
                // with the ring
                if (!mbar_wait(smem_u32(&dg_full), g & 1)) { ok = false; break; }
                mbar_expect_tx(smem_u32(&yr_full), 2u * (uint32_t)(te - tb) * C::TILE);
                for (int i = tb; i < te; ++i) {
                    tma_load_2d(smem_u32(smem + C::OFF_YR + (i - tb) * C::TILE), &tm_yr, 0,
                                (int32_t)(start + 128 * (int64_t)i), smem_u32(&yr_full));
                    // the B tiles again (their first copy was overwritten by G_lo)
                    tma_load_2d(smem_u32(smem + C::OFF_B2 + (i - tb) * C::TILE), &tm_b, 0,
                                (int32_t)(start + 128 * (int64_t)i), smem_u32(&yr_full));
                }
                ++yr_issued;
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
            if (b_issued > 0) mbar_wait(smem_u32(&b_full), (b_issued - 1) & 1);
            if (yr_issued > 0) mbar_wait(smem_u32(&yr_full), (yr_issued - 1) & 1);
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if (elect_one()) {
            constexpr Swz rsw = swz_for(C::RB);
            constexpr uint32_t id_q = idesc_bf16(128, C::M, false, false);   // B (K-major) . Wd1 (Wd1^T rows, K-major)
            constexpr uint32_t id_dg = idesc_bf16(128, C::M, false, false);  // dY (K-major) . Wd2 (K-major)
            constexpr uint32_t id_wt = idesc_bf16(128, C::WIDE ? 2 * C::M : C::M, true, true);   // dY^T (MN-major) . G (MN-major)
            constexpr uint32_t id_db = idesc_bf16(128, C::R, false, false);  // dQ (K-major) . Wd1^T (Wd1 rows, K-major)
            constexpr uint32_t id_w1 = idesc_bf16(128, C::M, true, true);    // B^T (MN-major) . dQ (MN-major)
            // shared-memory descriptors of slot / tile 0, advanced by adding the byte offset >> 4
            // to the start-address field (no carry: shared addresses < 256 KB). The 128-row B^T
            // operand has one real block of r rows: its block stride (LBO) is 0, so every block
            // reads the same r rows and the extra output rows are duplicates.
            const uint64_t yk0 = smem_desc(smem_u32(smem + C::OFF_Y), 16, 1024, kSwz128);     // dY, K-major
            const uint64_t ym0 = smem_desc(smem_u32(smem + C::OFF_Y), 16384, 1024, kSwz128);  // dY, MN-major
            const uint64_t wk0 = smem_desc(smem_u32(smem + C::OFF_W), 16, 1024, kSwz128);     // Wd2 slice
            // G, MN-major; WIDE: [G_hi | G_lo] as two N blocks (block stride = the hi -> lo distance)
            const uint64_t gm0 = smem_desc(smem_u32(smem + C::OFF_G), C::WIDE ? C::OFF_GLO - C::OFF_G : 0, 8 * C::RB, rsw);
            const uint64_t gl0 = smem_desc(smem_u32(smem + C::OFF_GLO), 0, 8 * C::RB, rsw);   // G_lo, MN-major
            const uint64_t bk0 = smem_desc(smem_u32(smem + C::OFF_B), 16, 8 * C::RB, rsw);    // B, K-major
            const uint64_t bm0 = smem_desc(smem_u32(smem + C::OFF_B2), 0, 8 * C::RB, rsw);    // B^T, MN-major (phase 2)
            const uint64_t qk0 = smem_desc(smem_u32(smem + C::OFF_DQ), 16, 8 * C::RB, rsw);   // dQ, K-major
            const uint64_t qm0 = smem_desc(smem_u32(smem + C::OFF_DQ), 0, 8 * C::RB, rsw);    // dQ, MN-major
            const uint64_t w1k = smem_desc(smem_u32(smem + C::OFF_WD1), 16, 8 * C::RB, rsw);  // Wd1 rows
            const uint64_t w1t = smem_desc(smem_u32(smem + C::OFF_WD1T), 16, 8 * C::RB, rsw); // Wd1^T rows
            constexpr uint64_t TILE16 = C::TILE >> 4;
            constexpr uint64_t KROWS16 = (16 * C::RB) >> 4;                 // 16 token rows of an r / m wide tile
            constexpr uint64_t LO16 = (C::OFF_DQLO - C::OFF_DQ) >> 4;       // dQ hi tile -> lo tile
            uint32_t yit = 0, wit = 0, cit = 0;
            bool ok = true;
            for (int g = 0; g < ngroups && ok; ++g) {
                int tb, te;
                group_tiles(g, ngroups, ntiles, tb, te);
                // TMEM of the previous group (dG / dB, Q, dWd1) has been read out
                if (g > 0) ok = mbar_wait(smem_u32(&dg_empty), (g - 1) & 1);
                ok = ok && mbar_wait(smem_u32(&b_full), g & 1);
                tc_fence_after();
                // ---- phase 0: Q_tile = B_tile . Wd1 (K = r) ----
                for (int i = tb; i < te && ok; ++i) {
                    const uint64_t bk = bk0 + (i - tb) * TILE16;
#pragma unroll
                    for (int k = 0; k < C::R / 16; ++k)
                        mma_bf16(tmem + C::TM_Q + (i - tb) * C::MS, bk + 2 * k, w1t + 2 * k, id_q, k > 0);
                }
                mma_commit(smem_u32(&q_full));
                // ---- phase 1: the dY stream ----
                for (int c = 0; c < nch && ok; ++c, ++cit) {
                    const uint32_t sw = wit % C::NW;
                    const uint32_t ab = cit % C::NWB;
                    ok = mbar_wait(smem_u32(&w_full[sw]), (wit / C::NW) & 1) &&
                         mbar_wait(smem_u32(&wt_empty[ab]), ((cit / C::NWB) & 1) ^ 1);
                    tc_fence_after();
                    const uint64_t wk = wk0 + ((sw * C::W_STAGE) >> 4);
                    const uint32_t d_wt = tmem + C::TM_WT + ab * C::MSW;
                    for (int i = tb; i < te && ok; ++i, ++yit) {
                        const int64_t t0 = start + 128 * (int64_t)i;
                        const int valid = (int)((end - t0) < 128 ? (end - t0) : 128);
                        const uint32_t s = yit % C::NSY;
                        ok = mbar_wait(smem_u32(&y_full[s]), (yit / C::NSY) & 1);
                        tc_fence_after();
                        if (!ok) break;   // a wait gave up: issue nothing more
                        const uint64_t yk = yk0 + ((s * C::Y_STAGE) >> 4);
                        const uint64_t ym = ym0 + ((s * C::Y_STAGE) >> 4);
                        const uint64_t gm = gm0 + (i - tb) * TILE16;
                        const uint64_t gl = gl0 + (i - tb) * TILE16;
                        const uint32_t d_dg = tmem + C::TM_DG + (i - tb) * C::MS;
                        // dG_tile += dY_tile . Wd2_chunk^T: K = 128 columns in 8 steps of 16
                        mma_bf16(d_dg, yk, wk, id_dg, c != 0);
#pragma unroll
                        for (int k = 1; k < 8; ++k)
                            mma_bf16(d_dg, yk + kmaj_off(k, 16384), wk + kmaj_off(k, C::M * 128), id_dg, true);
                        // the dWd2 product needs the tile's G (published per tile in phase 0,
                        // once per group; the dG products above did not wait for it)
                        if (c == 0) {
                            ok = ok && mbar_wait(smem_u32(&g_full[i - tb]), g & 1);
                            tc_fence_after();
                            if (!ok) break;
                        }
                        // dWd2T_chunk += dY_tile^T . (G_hi + G_lo)_tile: K = the tile's tokens in
                        // steps of 16
                        if (valid == 128) {
#pragma unroll
                            for (int k = 0; k < 8; ++k) {
                                mma_bf16(d_wt, ym + ((k * 2048) >> 4), gm + k * KROWS16, id_wt, (i > tb) || (k > 0));
                                if (!C::WIDE) mma_bf16(d_wt, ym + ((k * 2048) >> 4), gl + k * KROWS16, id_wt, true);
                            }
                        } else {
                            const int nks = (valid + 15) / 16;
                            for (int k = 0; k < nks; ++k) {
                                mma_bf16(d_wt, ym + ((k * 2048) >> 4), gm + k * KROWS16, id_wt, (i > tb) || (k > 0));
                                if (!C::WIDE) mma_bf16(d_wt, ym + ((k * 2048) >> 4), gl + k * KROWS16, id_wt, true);
                            }
                        }
                        mma_commit(smem_u32(&y_empty[s]));
                    }
                    mma_commit(smem_u32(&w_empty[sw]));
                    mma_commit(smem_u32(&wt_full[ab]));
                    ++wit;
                }
                mma_commit(smem_u32(&g_empty));
                mma_commit(smem_u32(&dg_full));
                // ---- phase 2: dB_tile = (dQ_hi + dQ_lo) . Wd1^T (K = m);
                //      dWd1 += B^T . (dQ_hi + dQ_lo) (K = tokens) ----
                ok = ok && mbar_wait(smem_u32(&yr_full), g & 1);   // the reloaded B tiles
                tc_fence_after();
                for (int i = tb; i < te && ok; ++i) {
                    const int64_t t0 = start + 128 * (int64_t)i;
                    const int valid = (int)((end - t0) < 128 ? (end - t0) : 128);
                    ok = mbar_wait(smem_u32(&dq_full[i - tb]), g & 1);
                    tc_fence_after();
                    if (!ok) break;
                    const uint64_t qk = qk0 + (i - tb) * TILE16;
                    const uint64_t qm = qm0 + (i - tb) * TILE16;
                    const uint64_t bm = bm0 + (i - tb) * TILE16;
                    const uint32_t d_db = tmem + C::TM_DG + (i - tb) * C::MS;
#pragma unroll
                    for (int k = 0; k < C::M / 16; ++k) mma_bf16(d_db, qk + 2 * k, w1k + 2 * k, id_db, k > 0);
#pragma unroll
                    for (int k = 0; k < C::M / 16; ++k) mma_bf16(d_db, qk + LO16 + 2 * k, w1k + 2 * k, id_db, true);
                    const int nks = (valid + 15) / 16;
                    for (int k = 0; k < nks; ++k) {
                        mma_bf16(tmem + C::TM_W1, bm + k * KROWS16, qm + k * KROWS16, id_w1, (i > tb) || (k > 0));
                        mma_bf16(tmem + C::TM_W1, bm + k * KROWS16, qm + LO16 + k * KROWS16, id_w1, true);
                    }
                    mma_commit(smem_u32(&db_full[i - tb]));
                }
                mma_commit(smem_u32(&w1_full));
            }
            mma_commit(smem_u32(&done_bar));
            mbar_wait(smem_u32(&done_bar), 0);
        }
    } else {
        // ---------------- epilogue warps ----------------
        const int q = warp & 3;
        const int row = q * 32 + lane;  // token row (phases 0, 2) or d-column row (phase 1)
        const int et = threadIdx.x - 64;
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        uint32_t cit = 0;
        bool ok = true;
        for (int g = 0; g < ngroups && ok; ++g) {
            int tb, te;
            group_tiles(g, ngroups, ntiles, tb, te);
            const int64_t slot = (int64_t)blockIdx.x * a.max_groups + g;
            // ---- phase 0: G = phi(Q) of every tile of the group ----
            ok = mbar_wait(smem_u32(&g_empty), (g & 1) ^ 1) && mbar_wait(smem_u32(&q_full), g & 1);
            tc_fence_after();
            for (int i = tb; i < te; ++i) {
                const int64_t t0 = start + 128 * (int64_t)i;
                const bool active = t0 + row < end;
                float v[C::M];
                tmem_ld_row<C::M>(tmem + lane_base + C::TM_Q + (i - tb) * C::MS, v);
                act_fast_row<C::M>(a.act, v);
#pragma unroll
                for (int j = 0; j < C::M; ++j) v[j] = active ? v[j] : 0.0f;
                store_bf16_swz_row<C::M>(smem + C::OFF_G + (i - tb) * C::TILE, row, v);
                // G_lo = G - bf16(G), over the tile's B rows (the Q products are done: q_full)
#pragma unroll
                for (int j = 0; j < C::M; ++j) v[j] -= __bfloat162float(__float2bfloat16_rn(v[j]));
                store_bf16_swz_row<C::M>(smem + C::OFF_GLO + (i - tb) * C::TILE, row, v);
                // publish this tile's G so its first dWd2 product can start
                fence_async_smem();
                named_barrier(1, 128);
                if (et == 0) mbar_arrive(smem_u32(&g_full[i - tb]));
            }

            // ---- phase 1: drain each chunk's dWd2^T partial ----
            // With a cluster exchange, the rows this CTA sends go out as soon as their chunk is
            // complete, and the rows it owns are read out at the start of the next chunk's turn
            // (the peers' rows of that chunk have arrived by then; the accumulator waits in TMEM).
            const bool defer = xg.exchanging() && xg.owns(row);
            int pend = -1, pend_cc = 0;
            // one row of a finished dWd2^T accumulator (WIDE: its hi part + its lo part)
            auto load_wt = [&](int buf, float (&v)[C::M]) {
                tmem_ld_row<C::M>(tmem + lane_base + C::TM_WT + buf * C::MSW, v);
                if (C::WIDE) {
                    float w[C::M];
                    tmem_ld_row<C::M>(tmem + lane_base + C::TM_WT + buf * C::MSW + C::M, w);
#pragma unroll
                    for (int j = 0; j < C::M; ++j) v[j] += w[j];
                }
            };
            auto drain_owned = [&](int buf, int chunk) {
                float v[C::M];
                load_wt(buf, v);
                tc_fence_before();
                mbar_arrive(smem_u32(&wt_empty[buf]));   // the accumulator is free again
                return xg.receive(a.wg, v, chunk, row, g == 0);
            };
            for (int c = 0; c < nch && ok; ++c, ++cit) {
                const int cc = c + c_first < nch ? c + c_first : c + c_first - nch;
                const uint32_t ab = cit % C::NWB;
                if (pend >= 0) {
                    ok = drain_owned(pend, pend_cc);
                    pend = -1;
                }
                ok = ok && mbar_wait(smem_u32(&wt_full[ab]), (cit / C::NWB) & 1);
                tc_fence_after();
                if (defer) {
                    pend = (int)ab;
                    pend_cc = cc;
                    continue;
                }
                float v[C::M];
                load_wt((int)ab, v);
                tc_fence_before();
                mbar_arrive(smem_u32(&wt_empty[ab]));   // the accumulator is free again
                if (xg.exchanging()) {
                    ok = ok && xg.send(v, row);
                } else {
                    xg.store_own(a.wg, v, cc, row, g == 0);
                }
            }
            if (ok && pend >= 0) ok = drain_owned(pend, pend_cc);   // the group's last chunk

            // ---- phase 2: dQ (hi + lo), then dB and the dWd1 partial ----
            ok = ok && mbar_wait(smem_u32(&dg_full), g & 1);
            tc_fence_after();
            for (int i = tb; i < te; ++i) {
                const int64_t t0 = start + 128 * (int64_t)i;
                const bool active = t0 + row < end;
                float hi[C::M], lo[C::M];
                tmem_ld_row<C::M>(tmem + lane_base + C::TM_DG + (i - tb) * C::MS, hi);
                tmem_ld_row<C::M>(tmem + lane_base + C::TM_Q + (i - tb) * C::MS, lo);
                dact_fast_row<C::M>(a.act, lo, lo);   // phi'(Q)
#pragma unroll
                for (int j = 0; j < C::M; ++j) {
                    const float x = active ? hi[j] * lo[j] : 0.0f;
                    hi[j] = __bfloat162float(__float2bfloat16_rn(x));
                    lo[j] = x - hi[j];
                }
                store_bf16_swz_row<C::M>(smem + C::OFF_DQ + (i - tb) * C::TILE, row, hi);
                store_bf16_swz_row<C::M>(smem + C::OFF_DQLO + (i - tb) * C::TILE, row, lo);
                // dG of the tile is read (its columns receive dB next) and dQ is published
                tc_fence_before();
                fence_async_smem();
                named_barrier(1, 128);
                if (et == 0) mbar_arrive(smem_u32(&dq_full[i - tb]));
            }
            ok = ok && mbar_wait(smem_u32(&yr_full), g & 1);
            for (int i = tb; i < te && ok; ++i) {
                const int64_t t0 = start + 128 * (int64_t)i;
                const bool active = t0 + row < end;
                ok = mbar_wait(smem_u32(&db_full[i - tb]), g & 1);
                tc_fence_after();
                float o[C::R];
                tmem_ld_row<C::R>(tmem + lane_base + C::TM_DG + (i - tb) * C::MS, o);
                if (active) {
                    // dB = [merge] dY[:, :r] + dQ . Wd1^T
                    if (a.merge) {
                        float y[C::R];
                        load_bf16_swz_row<C::R>(smem + C::OFF_YR + (i - tb) * C::TILE, row, y);
#pragma unroll
                        for (int e = 0; e < C::R; ++e) o[e] = y[e] + o[e];
                    }
                    uint4 *dbo = reinterpret_cast<uint4 *>(a.dB + (t0 + row) * C::R);
#pragma unroll
                    for (int v8 = 0; v8 < C::R / 8; ++v8) {
                        uint32_t pk[4];
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            __nv_bfloat162 hh = __floats2bfloat162_rn(o[8 * v8 + 2 * e], o[8 * v8 + 2 * e + 1]);
                            pk[e] = *reinterpret_cast<uint32_t *>(&hh);
                        }
                        dbo[v8] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
                    }
                }
            }
            // the group's dWd1 (rows = r, lanes 0 .. r-1) to its partial slot
            ok = ok && mbar_wait(smem_u32(&w1_full), g & 1);
            tc_fence_after();
            if (q * 32 < C::R) {
                float w[C::M];
                tmem_ld_row<C::M>(tmem + lane_base + C::TM_W1, w);
                if (row < C::R) {
                    float4 *dst = reinterpret_cast<float4 *>(a.part1 + (slot * C::R + row) * C::M);
#pragma unroll
                    for (int e = 0; e < C::M / 4; ++e) dst[e] = make_float4(w[4 * e], w[4 * e + 1], w[4 * e + 2], w[4 * e + 3]);
                }
            }
            tc_fence_before();
            mbar_arrive(smem_u32(&dg_empty));
            named_barrier(1, 128);   // phase-2 scratch reads done before the ring is reused
            if (et == 0) mbar_arrive(smem_u32(&p2_done));
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, C::TMEM_COLS);
    }
    if (C::CLMAX > 1 && xg.cl > 1) cluster_sync();   // no peer addresses this CTA's shared memory any more
    // Started without waiting for the previous kernel: wait for it now, so that this grid does
    // not complete before it (the kernels after this one wait for this grid only).
    if (a.after_independent) griddep_wait();
}

// out = sum over slots s = 0, 1, ... of part[s] (rows x cols each, rows * cols % 4 == 0), each
// element summed in slot order. Four consecutive elements per thread (16-byte loads), loaded in
// batches of eight slots, keep enough reads in flight. With transpose the result is written
// cols x rows (part slices are d x m, the weight gradient is m x d); out4 says out is 16-byte
// aligned (untransposed only).
__device__ __forceinline__ void add4(float4 &a, const float4 &b)
{
    a.x += b.x; a.y += b.y; a.z += b.z; a.w += b.w;
}

// Fixed-order sums of per-CTA partial fp32 matrices. A job sums `slots` matrices of rows x cols
// (rows * cols % 4 == 0) into `out` (transposed to cols x rows if `transpose`; `out4`: out is
// 16-byte aligned). A block of 32 x kSlotGroups threads owns 32 consecutive float4 columns of
// the flattened matrix; thread row g sums the g-th contiguous range of slots in slot order, and
// the groups' sums are then added in group order: the same order for every launch, so results
// are bitwise reproducible. One launch runs two jobs (the two weight gradients of a backward
// op): blocks [0, first.blocks) take the first, the rest the second.
constexpr int kSlotGroups = 8;

struct ReduceJob {
    const float *part;
    int64_t slots, rows, cols;
    float *out;
    int transpose, out4;
    int blocks;
};

__device__ __forceinline__ void reduce_job(const ReduceJob &j, int64_t block, int64_t nblocks, float4 (&grp)[kSlotGroups][32])
{
    const int64_t n4 = j.rows * j.cols / 4;
    const float4 *p4 = reinterpret_cast<const float4 *>(j.part);
    const int64_t per = (j.slots + kSlotGroups - 1) / kSlotGroups;
    const int64_t s0 = threadIdx.y * per;
    const int64_t s1 = s0 + per < j.slots ? s0 + per : j.slots;
    for (int64_t base = block * 32; base < n4; base += nblocks * 32) {
        const int64_t e4 = base + threadIdx.x;
        float4 acc = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
        if (e4 < n4) {
            // batches of eight slots, every load of a batch in flight before the first add
            for (int64_t s = s0; s < s1; s += 8) {
                float4 v[8];
#pragma unroll
                for (int u = 0; u < 8; ++u)
                    if (s + u < s1) v[u] = __ldcs(&p4[(s + u) * n4 + e4]);
#pragma unroll
                for (int u = 0; u < 8; ++u)
                    if (s + u < s1) add4(acc, v[u]);
            }
        }
        grp[threadIdx.y][threadIdx.x] = acc;
        __syncthreads();
        if (threadIdx.y == 0 && e4 < n4) {
            float4 t = grp[0][threadIdx.x];
#pragma unroll
            for (int g = 1; g < kSlotGroups; ++g) add4(t, grp[g][threadIdx.x]);
            const int64_t e = 4 * e4;
            if (j.transpose) {
                const int64_t rr = e / j.cols, cc = e - rr * j.cols;
                j.out[(cc + 0) * j.rows + rr] = t.x;
                j.out[(cc + 1) * j.rows + rr] = t.y;
                j.out[(cc + 2) * j.rows + rr] = t.z;
                j.out[(cc + 3) * j.rows + rr] = t.w;
            } else if (j.out4) {
                reinterpret_cast<float4 *>(j.out)[e4] = t;
            } else {
                j.out[e] = t.x; j.out[e + 1] = t.y; j.out[e + 2] = t.z; j.out[e + 3] = t.w;
            }
        }
        __syncthreads();
    }
}

__global__ void __launch_bounds__(32 * kSlotGroups) k_reduce_slots(const ReduceJob first, const ReduceJob second)
{
    __shared__ float4 grp[kSlotGroups][32];
    griddep_wait();
    griddep_launch_dependents();
    if ((int)blockIdx.x < first.blocks)
        reduce_job(first, blockIdx.x, first.blocks, grp);
    else
        reduce_job(second, blockIdx.x - first.blocks, gridDim.x - first.blocks, grp);
}

}  // namespace tc
}  // namespace resbm
