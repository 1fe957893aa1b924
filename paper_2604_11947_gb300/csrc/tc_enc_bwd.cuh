// tc_enc_bwd.cuh -- backward of the send side on tensor cores (chain rule of Sec. 3.2's encoder
// with the truncating identity path of Eq. Pid):
//   dA = dB . We2^T;  dP = dA * phi'(P);  dF = dP . We1^T;  dX[:, :r] += dB;
//   dWe1 = F^T . dP;  dWe2 = phi(P)^T . dB.
//
// Persistent CTAs (in clusters of 1, 2 or 4) over contiguous runs of whole 128-token tiles, in
// groups of up to NT tiles of 128 tokens. Every product runs on tcgen05; the CUDA cores apply
// phi and phi', convert, and do the identity-path update. For each group:
//   phase 0: the group's dB tiles (TMA) -> dA_tile = dB . We2^T in TMEM -> the epilogue reads P
//            (fp32, from the forward pass) and writes dP = dA * phi'(P) and A = phi(P) as bf16
//            rows [token][m] to shared memory (for m <= 32 dP also as hi + lo, hi = dP rounded
//            to bf16 and lo = the rounded remainder, so dF sees dP to about 16 significant
//            bits), and applies dX[:, :r] += dB -> dWe2 += A^T . dB over the group's tokens (the
//            A tile read MN-major as a 128-row operand whose rows >= m are never read back).
//            dB and A tiles live in F-ring slots 1 and 2, which the producer fills with F only
//            after phase 0.
//   phase 1: d in chunks of 128 columns; per chunk one We1 slice (128 x m, K-major) and per tile
//            one F tile (128 tokens x 128 columns) feeding
//              dF_tile_chunk (128 x 128 fp32, TMEM, double-buffered) = dP . We1_chunk^T
//              dWe1_chunk    (128 columns x m, TMEM, double-buffered) += F^T . dP
//            (F read MN-major, dP read K-major and MN-major). The epilogue converts dF to bf16
//            and stores it by TMA, and drains each finished dWe1 chunk into the cluster's fp32
//            partial slot (summed over the cluster's CTAs through distributed shared memory,
//            tc_wgrad.cuh); the group's dWe2 goes to its own per-CTA partial slot.
// Every CTA has the same number of tile groups (its tiles split evenly).
// HBM traffic per token: read F (2d), P (4m), dB (2r), dX[:, :r] (2r); write dF (2d),
// dX[:, :r] (2r). Per cluster: d x m fp32 partials; per CTA and group: m x r.
#pragma once

#include "common.cuh"
#include "tc_common.cuh"
#include "tc_wgrad.cuh"

namespace resbm {
namespace tc {

template <int M_> struct EncBwdCfg {
    static constexpr int M = M_;
    static constexpr int R = M_;
    static constexpr int MS = M_ < 32 ? 32 : M_;                 // TMEM columns per m-wide accumulator
    static constexpr int NT = M_ <= 32 ? 4 : 2;                  // tiles per group
    static constexpr int NSF = 3;                                // F ring depth
    static constexpr int NW = M_ <= 16 ? 4 : M_ <= 32 ? 2 : 3;   // We1 slice ring depth
    static constexpr int CLMAX = M_ <= 32 ? 4 : 1;               // CTAs per cluster (weight-gradient exchange)
    static constexpr int CL_MIN_TOKENS = 256;                 // clusters only from this many tokens per CTA
    static constexpr int NWB = CLMAX > 1 ? 3 : 2;                // dWe1 accumulators in TMEM
    static constexpr int NDA = M_ <= 32 ? NT : 1;                // dA TMEM regions (a ring)
    static constexpr bool DPLO = M_ <= 32;                       // dP kept as bf16 hi + lo for dF
    static constexpr uint32_t RB = M_ * 2;                       // row bytes (= swizzle) of r / m wide tiles
    static constexpr uint32_t F_STAGE = 128 * 128 * 2;
    static constexpr uint32_t STG_HALF = 128 * 64 * 2;           // dF staging: 128 rows x 64 columns
    static constexpr uint32_t W_STAGE = 128 * RB;                // We1 slice: 128 rows x m
    static constexpr uint32_t TILE = 128 * RB;                   // 128 tokens x r (or m) columns
    static constexpr uint32_t WE2_BYTES = M_ * R * 2;
    static constexpr uint32_t OFF_F = 0;
    static constexpr uint32_t OFF_STG = OFF_F + NSF * F_STAGE;
    static constexpr uint32_t OFF_W = OFF_STG + 2 * STG_HALF;
    static constexpr uint32_t OFF_DP = OFF_W + NW * W_STAGE;     // dP (hi) tiles [token][m]
    static constexpr uint32_t OFF_DPLO = OFF_DP + NT * TILE;     // dP lo tiles (if DPLO)
    static constexpr uint32_t OFF_WE2 = OFF_DPLO + (DPLO ? NT * TILE : 0);  // We2 [m][r], K-major
    static constexpr uint32_t OFF_RX = OFF_WE2 + WE2_BYTES;      // weight-gradient receive buffer
    static constexpr uint32_t SMEM_BYTES = OFF_RX + wgrad_rx_bytes<M_>(CLMAX) + 1024;
    // phase-0 scratch in F-ring slots 1 and 2
    static constexpr uint32_t OFF_DB = OFF_F + (NSF - 2) * F_STAGE;   // dB tiles [token][r] (TMA)
    static constexpr uint32_t OFF_A = OFF_F + (NSF - 1) * F_STAGE;    // A = phi(P) tiles [token][m]
    static_assert(NT * TILE <= F_STAGE && NSF >= 3, "phase-0 scratch must fit in two ring slots");
    static_assert(SMEM_BYTES <= 232448 - 512, "shared memory budget");
    // TMEM columns: dF 2 x 128 | dWe1 NWB x MS | dA NDA x MS | dWe2 MS
    static constexpr uint32_t TM_DF = 0, TM_WE = 256, TM_DA = 256 + NWB * MS, TM_W2 = TM_DA + NDA * MS;
    static_assert(TM_W2 + MS <= 512, "TMEM budget");
    static constexpr uint32_t TMEM_COLS = 512;
    static constexpr int THREADS = 192;
};

struct EncBwdArgs {
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
              const __grid_constant__ CUtensorMap tm_df16, const __grid_constant__ CUtensorMap tm_db,
              const EncBwdArgs a)
{
    using C = EncBwdCfg<M_>;
    griddep_wait();               // the previous kernel of the stream has completed
    griddep_launch_dependents();  // the next one may be scheduled on SMs as they free up
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    __shared__ uint64_t f_full[C::NSF], f_empty[C::NSF], w_full[C::NW], w_empty[C::NW];
    __shared__ uint64_t df_full[2], df_empty[2], we_full[C::NWB], we_empty[C::NWB];
    __shared__ uint64_t db_full, da_full[C::NDA], da_empty[C::NDA], dp_full[C::NT], p0_done, w2_full, st_done, done_bar;
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
        }
        for (int i = 0; i < C::NWB; ++i) {
            mbar_init(smem_u32(&we_full[i]), 1);
            mbar_init(smem_u32(&we_empty[i]), 128);
        }
        for (int i = 0; i < C::NDA; ++i) {
            mbar_init(smem_u32(&da_full[i]), 1);
            mbar_init(smem_u32(&da_empty[i]), 128);
        }
        for (int i = 0; i < C::NT; ++i) mbar_init(smem_u32(&dp_full[i]), 1);
        mbar_init(smem_u32(&db_full), 1);
        mbar_init(smem_u32(&p0_done), 2);   // the dWe2 MMAs' commit + the epilogue's dB reads
        mbar_init(smem_u32(&w2_full), 1);
        mbar_init(smem_u32(&st_done), 1);
        mbar_init(smem_u32(&done_bar), 1);
        xg.init_barriers();
        fence_mbar_init();
        xg.arm_first();
    }
    if (warp == 1) tmem_alloc(smem_u32(&tmem_base_sh), C::TMEM_COLS);
    if (warp >= 2) {  // We2 (m x r) as a swizzled K-major operand
        for (int e = threadIdx.x - 64; e < C::M * C::R; e += 128)
            *reinterpret_cast<__nv_bfloat16 *>(smem + C::OFF_WE2 + swz_offset(e / C::R, 2 * (e % C::R), C::RB)) = a.We2[e];
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
            tma_prefetch_desc(&tm_f128);
            tma_prefetch_desc(&tm_f16);
            tma_prefetch_desc(&tm_we1);
            tma_prefetch_desc(&tm_db);
            // F stages use slots 0, 1, ... from the start of every group (so that slots 1 and 2
            // can hold the phase-0 scratch); bit s of fpar is the fill count of slot s, mod 2
            uint32_t fpar = 0, filled = 0, wit = 0;
            int db_issued = 0;
            bool ok = true;
            for (int g = 0; g < ngroups && ok; ++g) {
                // the previous group's MMAs are done with the whole ring
                if (g > 0) ok = mbar_wait(smem_u32(&st_done), (g - 1) & 1);
                if (!ok) break;
                int tb, te;
                group_tiles(g, ngroups, ntiles, tb, te);
                mbar_expect_tx(smem_u32(&db_full), (uint32_t)(te - tb) * C::TILE);
                for (int i = tb; i < te; ++i)
                    tma_load_2d(smem_u32(smem + C::OFF_DB + (i - tb) * C::TILE), &tm_db, 0,
                                (int32_t)(start + 128 * (int64_t)i), smem_u32(&db_full));
                ++db_issued;
                bool p0_seen = false;
                uint32_t j = 0;   // F stage of this group
                for (int c = 0; c < nch && ok; ++c) {
                    const int cc = c + c_first < nch ? c + c_first : c + c_first - nch;
                    // order: F tile 0 of the chunk, the chunk's We1 slice, the other F tiles.
                    // The MMA needs the slice before any tile of the chunk, so it must not queue
                    // behind tiles that wait for ring slots (that would deadlock), and it must not
                    // delay the first tile (that would stall the stream on the small weight ring).
                    for (int i = tb; i < te; ++i) {
                        if (i == tb + 1) {
                            const uint32_t s = wit % C::NW;
                            if (!mbar_wait(smem_u32(&w_empty[s]), ((wit / C::NW) & 1) ^ 1)) { ok = false; break; }
                            mbar_expect_tx(smem_u32(&w_full[s]), C::W_STAGE);
                            tma_load_2d(smem_u32(smem + C::OFF_W + s * C::W_STAGE), &tm_we1, 0, cc * 128,
                                        smem_u32(&w_full[s]));
                            ++wit;
                        }
                        const int64_t t0 = start + 128 * (int64_t)i;
                        const int valid = (int)((end - t0) < 128 ? (end - t0) : 128);
                        const int nb = (valid + 15) / 16;
                        const uint32_t s = j % C::NSF;
                        if (s >= (uint32_t)(C::NSF - 2) && !p0_seen) {   // phase-0 scratch released
                            if (!mbar_wait(smem_u32(&p0_done), g & 1)) { ok = false; break; }
                            p0_seen = true;
                        }
                        if (!mbar_wait(smem_u32(&f_empty[s]), ((fpar >> s) & 1) ^ 1)) { ok = false; break; }
                        fpar ^= 1u << s;
                        filled |= 1u << s;
                        const uint32_t dst = smem_u32(smem + C::OFF_F + s * C::F_STAGE);
                        const uint32_t bar = smem_u32(&f_full[s]);
                        mbar_expect_tx(bar, valid == 128 ? C::F_STAGE : (uint32_t)nb * 2u * 2048u);
                        for (int h = 0; h < 2; ++h) {
                            if (valid == 128) {
                                tma_load_2d_hint(dst + h * 16384, &tm_f128, cc * 128 + 64 * h, (int32_t)t0, bar, stream_pol);
                            } else {
                                for (int rg = 0; rg < nb; ++rg)
                                    tma_load_2d_hint(dst + h * 16384 + rg * 2048, &tm_f16, cc * 128 + 64 * h,
                                                (int32_t)(t0 + 16 * rg), bar, stream_pol);
                            }
                        }
                        ++j;
                    }
                    if (!ok) break;
                    if (te - tb == 1) {  // a one-tile group: the slice after its only tile
                        const uint32_t s = wit % C::NW;
                        if (!mbar_wait(smem_u32(&w_empty[s]), ((wit / C::NW) & 1) ^ 1)) { ok = false; break; }
                        mbar_expect_tx(smem_u32(&w_full[s]), C::W_STAGE);
                        tma_load_2d(smem_u32(smem + C::OFF_W + s * C::W_STAGE), &tm_we1, 0, cc * 128,
                                    smem_u32(&w_full[s]));
                        ++wit;
                    }
                }
            }
            // drain the loads still in flight
            for (int s = 0; s < C::NSF; ++s)
                if ((filled >> s) & 1) mbar_wait(smem_u32(&f_full[s]), ((fpar >> s) & 1) ^ 1);
            for (uint32_t k = 0; k < (wit < (uint32_t)C::NW ? wit : (uint32_t)C::NW); ++k) {
                const uint32_t jj = wit - 1 - k;
                mbar_wait(smem_u32(&w_full[jj % C::NW]), (jj / C::NW) & 1);
            }
            if (db_issued > 0) mbar_wait(smem_u32(&db_full), (db_issued - 1) & 1);
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if (elect_one()) {
            constexpr Swz rsw = swz_for(C::RB);
            constexpr uint32_t id_da = idesc_bf16(128, C::M, false, false);   // dB (K-major) . We2 rows (K-major)
            constexpr uint32_t id_w2 = idesc_bf16(128, C::R, true, true);     // A^T (MN-major) . dB (MN-major)
            constexpr uint32_t id_df = idesc_bf16(128, 128, false, false);    // dP (K-major) . We1 (K-major)
            constexpr uint32_t id_we = idesc_bf16(128, C::M, true, true);     // F^T (MN-major) . dP (MN-major)
            // shared-memory descriptors of slot / tile 0, advanced by adding the byte offset >> 4
            // to the start-address field (no carry: shared addresses < 256 KB). The 128-row A^T
            // operand has one real block of m rows: its block stride (LBO) is 0, so every block
            // reads the same m rows and the extra output rows are duplicates.
            const uint64_t fm0 = smem_desc(smem_u32(smem + C::OFF_F), 16384, 1024, kSwz128);   // F, MN-major
            const uint64_t wd0 = smem_desc(smem_u32(smem + C::OFF_W), 16, 8 * C::RB, rsw);     // We1 slice
            const uint64_t pk0 = smem_desc(smem_u32(smem + C::OFF_DP), 16, 8 * C::RB, rsw);    // dP, K-major
            const uint64_t pm0 = smem_desc(smem_u32(smem + C::OFF_DP), 0, 8 * C::RB, rsw);     // dP, MN-major
            const uint64_t dbk0 = smem_desc(smem_u32(smem + C::OFF_DB), 16, 8 * C::RB, rsw);   // dB, K-major
            const uint64_t dbm0 = smem_desc(smem_u32(smem + C::OFF_DB), 0, 8 * C::RB, rsw);    // dB, MN-major
            const uint64_t am0 = smem_desc(smem_u32(smem + C::OFF_A), 0, 8 * C::RB, rsw);      // A^T, MN-major
            const uint64_t we2k = smem_desc(smem_u32(smem + C::OFF_WE2), 16, 8 * C::RB, rsw);  // We2 rows
            constexpr uint64_t TILE16 = C::TILE >> 4;
            constexpr uint64_t KROWS16 = (16 * C::RB) >> 4;              // 16 token rows of an r / m wide tile
            constexpr uint64_t LO16 = (C::OFF_DPLO - C::OFF_DP) >> 4;    // dP hi tile -> lo tile
            uint32_t fpar = 0, wit = 0, cit = 0, dfit = 0, u = 0;
            bool ok = true;
            for (int g = 0; g < ngroups && ok; ++g) {
                int tb, te;
                group_tiles(g, ngroups, ntiles, tb, te);
                ok = mbar_wait(smem_u32(&db_full), g & 1);
                tc_fence_after();
                // ---- phase 0: dA_tile = dB_tile . We2^T (K = r), a ring of NDA TMEM regions ----
                for (int i = tb; i < te && ok; ++i, ++u) {
                    const uint32_t rg = u % C::NDA;
                    if (u >= (uint32_t)C::NDA) {
                        ok = mbar_wait(smem_u32(&da_empty[rg]), ((u / C::NDA) - 1) & 1);
                        tc_fence_after();
                    }
                    const uint64_t dbk = dbk0 + (i - tb) * TILE16;
#pragma unroll
                    for (int k = 0; k < C::R / 16; ++k)
                        mma_bf16(tmem + C::TM_DA + rg * C::MS, dbk + 2 * k, we2k + 2 * k, id_da, k > 0);
                    mma_commit(smem_u32(&da_full[rg]));
                }
                // dWe2 += A_tile^T . dB_tile (K = the tile's tokens), once the tile's A is written
                for (int i = tb; i < te && ok; ++i) {
                    const int64_t t0 = start + 128 * (int64_t)i;
                    const int valid = (int)((end - t0) < 128 ? (end - t0) : 128);
                    ok = mbar_wait(smem_u32(&dp_full[i - tb]), g & 1);
                    tc_fence_after();
                    if (!ok) break;   // a wait gave up: issue nothing more
                    const uint64_t am = am0 + (i - tb) * TILE16;
                    const uint64_t dbm = dbm0 + (i - tb) * TILE16;
                    const int nks = (valid + 15) / 16;
                    for (int k = 0; k < nks; ++k)
                        mma_bf16(tmem + C::TM_W2, am + k * KROWS16, dbm + k * KROWS16, id_w2, (i > tb) || (k > 0));
                }
                mma_commit(smem_u32(&p0_done));   // dB and A tiles are no longer read
                mma_commit(smem_u32(&w2_full));
                // ---- phase 1: the F stream ----
                uint32_t j = 0;
                for (int c = 0; c < nch && ok; ++c, ++cit, ++wit) {
                    const uint32_t sw = wit % C::NW, ae = cit % C::NWB;
                    ok = mbar_wait(smem_u32(&w_full[sw]), (wit / C::NW) & 1) &&
                         mbar_wait(smem_u32(&we_empty[ae]), ((cit / C::NWB) & 1) ^ 1);
                    tc_fence_after();
                    if (!ok) break;
                    const uint64_t wd = wd0 + ((sw * C::W_STAGE) >> 4);
                    const uint32_t d_we = tmem + C::TM_WE + ae * C::MS;
                    for (int i = tb; i < te && ok; ++i, ++dfit, ++j) {
                        const int64_t t0 = start + 128 * (int64_t)i;
                        const int valid = (int)((end - t0) < 128 ? (end - t0) : 128);
                        const uint32_t s = j % C::NSF, ad_buf = dfit & 1;
                        ok = mbar_wait(smem_u32(&f_full[s]), (fpar >> s) & 1) &&
                             mbar_wait(smem_u32(&df_empty[ad_buf]), ((dfit >> 1) & 1) ^ 1);
                        fpar ^= 1u << s;
                        tc_fence_after();
                        if (!ok) break;
                        const uint64_t fm = fm0 + ((s * C::F_STAGE) >> 4);
                        const uint64_t pk = pk0 + (i - tb) * TILE16;
                        const uint64_t pm = pm0 + (i - tb) * TILE16;
                        const uint32_t d_df = tmem + C::TM_DF + ad_buf * 128;
                        // dF = dP . We1_chunk^T (K = m in steps of 16 = 32 bytes of a swizzled row)
#pragma unroll
                        for (int k = 0; k < C::M / 16; ++k) mma_bf16(d_df, pk + 2 * k, wd + 2 * k, id_df, k > 0);
                        if (C::DPLO) {
#pragma unroll
                            for (int k = 0; k < C::M / 16; ++k) mma_bf16(d_df, pk + LO16 + 2 * k, wd + 2 * k, id_df, true);
                        }
                        mma_commit(smem_u32(&df_full[ad_buf]));
                        // dWe1^T_chunk += F^T . dP  (K = the tile's tokens in steps of 16)
                        if (valid == 128) {
#pragma unroll
                            for (int k = 0; k < 8; ++k)
                                mma_bf16(d_we, fm + ((k * 2048) >> 4), pm + k * KROWS16, id_we, (i > tb) || (k > 0));
                        } else {
                            const int nks = (valid + 15) / 16;
                            for (int k = 0; k < nks; ++k)
                                mma_bf16(d_we, fm + ((k * 2048) >> 4), pm + k * KROWS16, id_we, (i > tb) || (k > 0));
                        }
                        mma_commit(smem_u32(&f_empty[s]));
                    }
                    mma_commit(smem_u32(&w_empty[sw]));
                    mma_commit(smem_u32(&we_full[ae]));
                }
                mma_commit(smem_u32(&st_done));
            }
            mma_commit(smem_u32(&done_bar));
            mbar_wait(smem_u32(&done_bar), 0);
        }
    } else {
        // ---------------- epilogue warps ----------------
        const int q = warp & 3;
        const int row = q * 32 + lane;
        const int et = threadIdx.x - 64;
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        uint32_t cit = 0, dfit = 0, sit = 0, u = 0;
        bool ok = true;
        for (int g = 0; g < ngroups && ok; ++g) {
            int tb, te;
            group_tiles(g, ngroups, ntiles, tb, te);
            const int64_t slot = (int64_t)blockIdx.x * a.max_groups + g;
            // ---- phase 0: dP and A = phi(P) of every tile, dX[:, :r] += dB ----
            // the group's P rows and dX[:, :r] rows towards L2 first, so that the per-tile loads
            // below do not each wait for DRAM
            for (int i = tb; i < te; ++i) {
                const int64_t tok = start + 128 * (int64_t)i + row;
                if (tok < end) {
                    prefetch_l2(a.P + tok * C::M);
                    if (C::M * 4 > 128) prefetch_l2(a.P + tok * C::M + 32);
                    if (a.dX) prefetch_l2(a.dX + tok * a.d);
                }
            }
            ok = mbar_wait(smem_u32(&db_full), g & 1);
            for (int i = tb; i < te; ++i, ++u) {
                const int64_t t0 = start + 128 * (int64_t)i;
                const bool active = t0 + row < end;
                const int64_t tok = t0 + row;
                // this token's P row and dX[:, :r] row, fetched before waiting for dA
                float pv[C::M];
                float xv[C::R];
#pragma unroll
                for (int jj = 0; jj < C::M; ++jj) pv[jj] = 0.0f;
#pragma unroll
                for (int jj = 0; jj < C::R; ++jj) xv[jj] = 0.0f;
                if (active) {
                    const float4 *ps = reinterpret_cast<const float4 *>(a.P + tok * C::M);
#pragma unroll
                    for (int jj = 0; jj < C::M / 4; ++jj) {
                        const float4 v = ps[jj];
                        pv[4 * jj] = v.x; pv[4 * jj + 1] = v.y; pv[4 * jj + 2] = v.z; pv[4 * jj + 3] = v.w;
                    }
                    if (a.dX) load_bf16_row<C::R>(a.dX + tok * a.d, xv);
                }
                const uint32_t rg = u % C::NDA;
                ok = ok && mbar_wait(smem_u32(&da_full[rg]), (u / C::NDA) & 1);
                tc_fence_after();
                float da[C::M];
                tmem_ld_row<C::M>(tmem + lane_base + C::TM_DA + rg * C::MS, da);
                tc_fence_before();
                mbar_arrive(smem_u32(&da_empty[rg]));   // the dA region is free again
                float av[C::M], dph[C::M];
                act_dact_fast_row<C::M>(a.act, pv, av, dph);
#pragma unroll
                for (int jj = 0; jj < C::M; ++jj) {
                    const float x = active ? da[jj] * dph[jj] : 0.0f;
                    da[jj] = __bfloat162float(__float2bfloat16_rn(x));   // hi
                    pv[jj] = x - da[jj];                                 // lo
                    av[jj] = active ? av[jj] : 0.0f;
                }
                store_bf16_swz_row<C::M>(smem + C::OFF_DP + (i - tb) * C::TILE, row, da);
                if (C::DPLO) store_bf16_swz_row<C::M>(smem + C::OFF_DPLO + (i - tb) * C::TILE, row, pv);
                store_bf16_swz_row<C::M>(smem + C::OFF_A + (i - tb) * C::TILE, row, av);
                // identity path: dX[:, :r] += dB
                if (active && a.dX) {
                    float db[C::R];
                    load_bf16_swz_row<C::R>(smem + C::OFF_DB + (i - tb) * C::TILE, row, db);
                    uint4 *xp = reinterpret_cast<uint4 *>(a.dX + tok * a.d);
#pragma unroll
                    for (int v8 = 0; v8 < C::R / 8; ++v8) {
                        uint32_t pk[4];
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            __nv_bfloat162 h = __floats2bfloat162_rn(xv[8 * v8 + 2 * e] + db[8 * v8 + 2 * e],
                                                                     xv[8 * v8 + 2 * e + 1] + db[8 * v8 + 2 * e + 1]);
                            pk[e] = *reinterpret_cast<uint32_t *>(&h);
                        }
                        xp[v8] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
                    }
                }
                // publish this tile's dP and A; after the last tile every thread's dB reads are
                // done (p0_done before the last dp_full, so the stream cannot overtake it)
                fence_async_smem();
                named_barrier(1, 128);
                if (et == 0) {
                    if (i == te - 1) mbar_arrive(smem_u32(&p0_done));
                    mbar_arrive(smem_u32(&dp_full[i - tb]));
                }
            }

            // ---- phase 1: dF tiles out by TMA; dWe1 chunks to the partial slot ----
            // With a cluster exchange, the rows this CTA sends go out as soon as their chunk is
            // complete, and the rows it owns are read out after the next chunk's first dF tile
            // (the peers' rows of that chunk have arrived by then; the accumulator waits in TMEM).
            const bool defer = xg.exchanging() && xg.owns(row);
            int pend = -1, pend_cc = 0;
            auto drain_owned = [&](int buf, int chunk) {
                float v[C::M];
                tmem_ld_row<C::M>(tmem + lane_base + C::TM_WE + buf * C::MS, v);
                tc_fence_before();
                mbar_arrive(smem_u32(&we_empty[buf]));   // the accumulator is free again
                return xg.receive(a.wg, v, chunk, row, g == 0);
            };
            for (int c = 0; c < nch && ok; ++c, ++cit) {
                const int cc = c + c_first < nch ? c + c_first : c + c_first - nch;
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
                        float v2[2][32];
                        if (gqend) {   // the half's 64 columns, both TMEM loads in flight
                            tmem_ld32(tmem + lane_base + C::TM_DF + ad_buf * 128 + h * 64, v2[0]);
                            tmem_ld32(tmem + lane_base + C::TM_DF + ad_buf * 128 + h * 64 + 32, v2[1]);
                            tmem_ld_wait();
                            tmem_regs_ready(v2[0]);
                            tmem_regs_ready(v2[1]);
                        }
#pragma unroll
                        for (int gq = 0; gq < 2; ++gq) {
                            if (gq >= gqend) break;
                            float (&v)[32] = v2[gq];
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
                            const int x = cc * 128 + 64 * h;
                            if (valid == 128) {
                                tma_store_2d_hint(&tm_df128, x, (int32_t)t0, smem_u32(stg), l2_evict_first());
                            } else {
                                for (int rgi = 0; rgi * 16 < valid; ++rgi)
                                    tma_store_2d_hint(&tm_df16, x, (int32_t)(t0 + 16 * rgi), smem_u32(stg) + rgi * 2048, l2_evict_first());
                            }
                            bulk_commit();
                        }
                    }
                    if (i == tb && pend >= 0) {
                        ok = ok && drain_owned(pend, pend_cc);
                        pend = -1;
                    }
                }
                // the chunk's dWe1 rows (lane = d column) -> the cluster's partial slot
                const uint32_t ae = cit % C::NWB;
                ok = ok && mbar_wait(smem_u32(&we_full[ae]), (cit / C::NWB) & 1);
                tc_fence_after();
                if (defer) {
                    pend = (int)ae;
                    pend_cc = cc;
                    continue;
                }
                float v[C::M];
                tmem_ld_row<C::M>(tmem + lane_base + C::TM_WE + ae * C::MS, v);
                tc_fence_before();
                mbar_arrive(smem_u32(&we_empty[ae]));   // the accumulator is free again
                if (xg.exchanging()) {
                    ok = ok && xg.send(v, row);
                } else {
                    xg.store_own(a.wg, v, cc, row, g == 0);
                }
            }
            if (ok && pend >= 0) ok = drain_owned(pend, pend_cc);   // the group's last chunk

            // ---- the group's dWe2 (rows = m, lanes 0 .. m-1) to its partial slot ----
            ok = ok && mbar_wait(smem_u32(&w2_full), g & 1);
            tc_fence_after();
            if (q * 32 < C::M) {
                float w[C::R];
                tmem_ld_row<C::R>(tmem + lane_base + C::TM_W2, w);
                if (row < C::M) {
                    float4 *dst = reinterpret_cast<float4 *>(a.part2 + (slot * C::M + row) * C::R);
#pragma unroll
                    for (int e = 0; e < C::R / 4; ++e) dst[e] = make_float4(w[4 * e], w[4 * e + 1], w[4 * e + 2], w[4 * e + 3]);
                }
            }
            tc_fence_before();
        }
        if (et == 0) bulk_wait<0>();
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, C::TMEM_COLS);
    }
    if (C::CLMAX > 1 && xg.cl > 1) cluster_sync();   // no peer addresses this CTA's shared memory any more
}

}  // namespace tc
}  // namespace resbm
