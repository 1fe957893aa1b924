// tc_dec_fwd.cuh -- receive side of the boundary on tensor cores (Sec. 3.2 decoder, Eq. Pid
// zero-padding identity path):  Y = [merge] B . I_{r x d} + phi(B . Wd1) . Wd2.
//
// Persistent CTAs. The work is cut in units of (128-token tile, NCH output columns) and every
// CTA owns a contiguous run of floor or ceil(units / grid) of them in tile-major order: one
// segment of consecutive chunks per tile it touches (the tiles at the ends of its run partly).
// Y's columns are independent given G, so no tile has to be finished by one CTA and the runs
// balance to within one chunk. Per segment:
//   producer warp  : the tile's B rows by TMA (double-buffered; the next tile's as soon as its
//                    buffer is free); Wd2 column chunks (m x NCH, MN-major) into a ring
//   MMA warp       : Q = B . Wd1 of the NEXT segment's tile one chunk before this segment's
//                    last, then per chunk D_chunk (128 x NCH fp32, TMEM, double-buffered) =
//                    G . Wd2_chunk; with G double-buffered the epilogue computes the next tile's
//                    G while this tile's last chunk is being computed (no bubble between tiles)
//   epilogue warps : G = phi(Q) -> bf16 -> shared memory (the A operand, K-major), then per
//                    chunk TMEM -> registers, + B on the first r columns (chunk 0 only), -> bf16
//                    -> swizzled staging -> TMA store of Y (boxes of 128 rows, or 16 rows for a
//                    partial tile). Eight warps, two per TMEM lane quarter, each pair splitting
//                    a chunk's columns: one warp's TMEM and shared-memory latencies overlap the
//                    other's work (with one warp per quarter the epilogue set the pace).
// HBM traffic per token: read B (2r bytes, once per segment), write Y (2d bytes); Wd2 is
// re-read from L2.
//
// The next block's pre-attention RMSNorm fused in (NORM): N = Y / sqrt(mean_j Y_j^2 + eps) * gamma
// with Y as stored (bf16) needs a row's sum of squares over all d columns before any of its N
// values, and a row's chunks may lie in several CTAs. So the kernel runs twice on the same B:
//   NORM = 1 stores Y and, per row, chunk and column half, the sum of squares of the stored
//            (rounded) Y values into the slot ss[2 c + half][token] (fp32; the even and the odd
//            columns summed separately in column order, then added);
//   k_row_rstd sums each row's 2 d / NCH slots in slot order: rstd = 1 / sqrt(sum / d + eps),
//            and writes gamma as fp32;
//   NORM = 2 recomputes the same fp32 values (same products, same order) and stores
//            N = bf16((y * rstd) * gamma) instead of Y, y the fp32 value that rounds to the stored
//            Y (paired fp32 multiplies, each rounded as a single one). Against the norm of the
//            stored Y this skips one rounding of y: N differs from it by less than half Y's
//            spacing times rstd * gamma before N's own rounding (and is closer to the exact norm).
// Y never travels back from memory: per token the three launches read 2 x 2r bytes of B and
// 8 d / NCH + 4 bytes of sums and write Y and N (4d bytes), against 6d for a separate norm over a
// stored Y.
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
    static constexpr uint32_t GB = M_ * 2 < 128 ? M_ * 2 : 128;   // row bytes (= swizzle) of a 128-row block
    static constexpr int NB = M_ * 2 / GB;             // such blocks across the r (or m) columns
    static constexpr int SPB = GB / 32;                // 16-element K steps per block
    static constexpr uint32_t W_STAGE_BYTES = M_ * NCH * 2;
    static constexpr uint32_t TILE_BYTES = 128 * M_ * 2;   // 128 tokens x r (or m) bf16, NB blocks
    static constexpr uint32_t STG_BYTES = 128 * NCH * 2;
    static constexpr uint32_t WD1T_BYTES = R * M_ * 2;
    // shared-memory map (offsets from a 1024-aligned base)
    static constexpr uint32_t OFF_W = 0;
    // G and B tiles double-buffered (the next tile's G is made while this tile's last chunk is
    // computed) where shared memory allows, i.e. for m <= 64
    static constexpr int NGB = M_ <= 64 ? 2 : 1;
    static constexpr bool LOOKAHEAD = NGB == 2;
    static constexpr uint32_t OFF_G = OFF_W + NSTAGE * W_STAGE_BYTES;   // NGB G tiles [token][m]
    static constexpr uint32_t OFF_B = OFF_G + NGB * TILE_BYTES;          // NGB B tiles [token][r] (TMA)
    static constexpr uint32_t OFF_STG = OFF_B + NGB * TILE_BYTES;
    static constexpr uint32_t OFF_WD1T = OFF_STG + 2 * STG_BYTES;       // Wd1^T [m][r], K-major
    static constexpr uint32_t SMEM_BYTES = OFF_WD1T + WD1T_BYTES + 1024;  // + alignment slack
    static_assert(SMEM_BYTES <= 232448 - 512, "shared memory budget");
    static constexpr uint32_t TMEM_COLS = 2 * NCH;
    static constexpr int EPI = 256;                    // epilogue threads (8 warps)
    static constexpr int THREADS = 64 + EPI;
};

struct DecFwdArgs {
    const __nv_bfloat16 *Wd1;   // r x m
    int64_t T, d;
    int act, merge;
    float *ss;                    // NORM = 1: 2 d / NCH slots x T row sums of squares
    const float *rstd;            // NORM = 2: T reciprocal row RMS (k_row_rstd)
    const float *gamma;           // NORM = 2: the norm's weight (d, fp32, 16-byte aligned)
};

// rstd[t] = 1 / sqrt(sum of the row's nslots partial sums of squares, in slot order, / d + eps);
// gamma32 = gamma as fp32
__global__ void __launch_bounds__(256) k_row_rstd(const float *__restrict__ ss, int nslots, int64_t T, int64_t d,
                                                  float eps, float *__restrict__ rstd,
                                                  const __nv_bfloat16 *__restrict__ gamma, float *__restrict__ gamma32)
{
    griddep_wait();
    griddep_launch_dependents();
    const int64_t n = T > d ? T : d;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < n; t += (int64_t)gridDim.x * blockDim.x) {
        if (t < d) gamma32[t] = __bfloat162float(gamma[t]);
        if (t < T) {
            // eight slots' loads in flight at a time, added in slot order
            float sq = 0.0f;
            int sl = 0;
            for (; sl + 8 <= nslots; sl += 8) {
                float x[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) x[u] = ss[(int64_t)(sl + u) * T + t];
#pragma unroll
                for (int u = 0; u < 8; ++u) sq += x[u];
            }
            for (; sl < nslots; ++sl) sq += ss[(int64_t)sl * T + t];
            rstd[t] = 1.0f / sqrtf(sq / (float)d + eps);
        }
    }
}

// Receive side. Per tile of 128 tokens: the producer loads the tile's B rows by TMA; the MMA
// computes Q = B . Wd1 into the next free accumulator (a "chunk" of its own in the accumulator
// sequence); the epilogue turns Q into G = phi(Q) (bf16, shared memory) and then drains the
// tile's Y chunks (G . Wd2_chunk, + B on the first r columns), storing them by TMA.
template <int M_, int NORM = 0>
__global__ void __launch_bounds__(320, 1)
    k_dec_fwd(const __grid_constant__ CUtensorMap tm_wd2, const __grid_constant__ CUtensorMap tm_y128,
              const __grid_constant__ CUtensorMap tm_y16, const __grid_constant__ CUtensorMap tm_b,
              const DecFwdArgs a)
{
    using C = DecFwdCfg<M_>;
    static_assert(NORM >= 0 && NORM <= 2, "0: Y; 1: Y and row sums of squares; 2: the normalised rows");
    griddep_wait();               // the previous kernel of the stream has completed
    griddep_launch_dependents();  // the next one may be scheduled on SMs as they free up
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    __shared__ uint64_t w_full[C::NSTAGE], w_empty[C::NSTAGE];
    __shared__ uint64_t b_full[C::NGB], b_empty[C::NGB], g_full[C::NGB], acc_full[2], acc_empty[2], done_bar;
    __shared__ uint32_t tmem_base_sh;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nchunks = (int)(a.d / C::NCH);   // d % NCH == 0 on this path
    // this CTA's run of (tile, chunk) units
    const int64_t units = ((a.T + 127) / 128) * nchunks;
    const int64_t u_begin = units * blockIdx.x / gridDim.x, u_end = units * (blockIdx.x + 1) / gridDim.x;
    // segment k of the run: tile, first and one-past-last chunk
    auto seg_at = [&](int64_t u, int64_t &tile, int &c0, int &c1) {
        tile = u / nchunks;
        c0 = (int)(u - tile * nchunks);
        const int64_t last = u_end - tile * nchunks;
        c1 = last < nchunks ? (int)last : nchunks;
    };

    if (threadIdx.x == 0) {
        for (int s = 0; s < C::NSTAGE; ++s) {
            mbar_init(smem_u32(&w_full[s]), 1);
            mbar_init(smem_u32(&w_empty[s]), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(smem_u32(&acc_full[i]), 1);
            mbar_init(smem_u32(&acc_empty[i]), C::EPI);
        }
        for (int i = 0; i < C::NGB; ++i) {
            mbar_init(smem_u32(&b_full[i]), 1);
            mbar_init(smem_u32(&b_empty[i]), 1);
            mbar_init(smem_u32(&g_full[i]), 1);
        }
        mbar_init(smem_u32(&done_bar), 1);
        fence_mbar_init();
    }
    if (warp == 1) tmem_alloc(smem_u32(&tmem_base_sh), C::TMEM_COLS);
    if (warp >= 2) {  // Wd1^T (m x r) as a swizzled K-major operand: NB blocks of GB-byte rows
        for (int e = threadIdx.x - 64; e < C::R * C::M; e += C::EPI) {
            const int k = e / C::M, n = e % C::M;   // Wd1[k][n]
            const int kb = k / (C::GB / 2), kk = k % (C::GB / 2);
            *reinterpret_cast<__nv_bfloat16 *>(smem + C::OFF_WD1T + kb * (C::M * C::GB) + swz_offset(n, 2 * kk, C::GB)) =
                a.Wd1[e];
        }
        fence_async_smem();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_base_sh;

    if (warp == 0) {
        // ---------------- producer: B tiles and Wd2 chunks ----------------
        if (elect_one()) {
            tma_prefetch_desc(&tm_wd2);
            tma_prefetch_desc(&tm_b);
            // B rows of segment k's tile into buffer k % NGB, once that buffer's previous tile is
            // no longer read (128-row boxes: rows past T read as zeros)
            auto load_b = [&](uint32_t k, int64_t tile) -> bool {
                const uint32_t bb = k % C::NGB;
                if (!mbar_wait(smem_u32(&b_empty[bb]), ((k / C::NGB) & 1) ^ 1)) return false;
                mbar_expect_tx(smem_u32(&b_full[bb]), C::TILE_BYTES);
                for (int b = 0; b < C::NB; ++b)
                    tma_load_2d(smem_u32(smem + C::OFF_B + bb * C::TILE_BYTES + b * (128 * C::GB)), &tm_b,
                                b * (C::GB / 2), (int32_t)(tile * 128), smem_u32(&b_full[bb]));
                return true;
            };
            uint32_t it = 0, k = 0, b_loaded = 0;
            bool ok = true;
            if (u_begin < u_end) {
                int64_t tile;
                int c0, c1;
                seg_at(u_begin, tile, c0, c1);
                ok = load_b(0, tile);
                b_loaded = ok ? 1 : 0;
            }
            for (int64_t u = u_begin; u < u_end && ok; ++k) {
                int64_t tile;
                int c0, c1;
                seg_at(u, tile, c0, c1);
                u = tile * nchunks + c1;
                if (C::LOOKAHEAD && u < u_end) {   // the next segment's B, early: its Q comes before this one's end
                    int64_t nt;
                    int n0, n1;
                    seg_at(u, nt, n0, n1);
                    if (!(ok = load_b(k + 1, nt))) break;
                    ++b_loaded;
                }
                for (int c = c0; c < c1; ++c) {
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
                if (!C::LOOKAHEAD && ok && u < u_end) {   // one B buffer: the next tile's after this segment's chunks
                    int64_t nt;
                    int n0, n1;
                    seg_at(u, nt, n0, n1);
                    if (!(ok = load_b(k + 1, nt))) break;
                    ++b_loaded;
                }
            }
            // drain: every issued load has landed before the CTA can exit
            const uint32_t n = it < (uint32_t)C::NSTAGE ? it : (uint32_t)C::NSTAGE;
            for (uint32_t j0 = 0; j0 < n; ++j0) {
                const uint32_t j = it - 1 - j0;
                mbar_wait(smem_u32(&w_full[j % C::NSTAGE]), (j / C::NSTAGE) & 1);
            }
            for (uint32_t j0 = 0; j0 < (b_loaded < (uint32_t)C::NGB ? b_loaded : (uint32_t)C::NGB); ++j0) {
                const uint32_t j = b_loaded - 1 - j0;
                mbar_wait(smem_u32(&b_full[j % C::NGB]), (j / C::NGB) & 1);
            }
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if (elect_one()) {
            constexpr Swz gsw = swz_for(C::GB);
            constexpr uint32_t id_q = idesc_bf16(128, C::M, false, false);    // B (K-major) . Wd1^T rows (K-major)
            constexpr uint32_t id_y = idesc_bf16(128, C::NCH, false, true);   // G (K-major) . Wd2 chunk (MN-major)
            constexpr uint64_t TILE16 = C::TILE_BYTES >> 4;
            const uint64_t bk0 = smem_desc(smem_u32(smem + C::OFF_B), 16, 8 * C::GB, gsw);
            const uint64_t gk0 = smem_desc(smem_u32(smem + C::OFF_G), 16, 8 * C::GB, gsw);
            const uint64_t wt0 = smem_desc(smem_u32(smem + C::OFF_WD1T), 16, 8 * C::GB, gsw);
            uint32_t it = 0, acc_it = 0;
            bool ok = true;
            // Q = B . Wd1 of segment k's tile (B buffer k % NGB) into the next accumulator
            auto issue_q = [&](uint32_t k) {
                const uint32_t ab = acc_it & 1;
                ok = ok && mbar_wait(smem_u32(&b_full[k % C::NGB]), (k / C::NGB) & 1) &&
                     mbar_wait(smem_u32(&acc_empty[ab]), ((acc_it >> 1) & 1) ^ 1);
                tc_fence_after();
                if (!ok) return;
#pragma unroll
                for (int kk = 0; kk < C::R / 16; ++kk) {
                    const uint64_t off = (uint64_t)(((kk / C::SPB) * (128 * C::GB) + (kk % C::SPB) * 32) >> 4);
                    const uint64_t woff = (uint64_t)(((kk / C::SPB) * (C::M * C::GB) + (kk % C::SPB) * 32) >> 4);
                    mma_bf16(tmem + ab * C::NCH, bk0 + (k % C::NGB) * TILE16 + off, wt0 + woff, id_q, kk > 0);
                }
                mma_commit(smem_u32(&acc_full[ab]));
                ++acc_it;
            };
            if (u_begin < u_end) issue_q(0);
            uint32_t k = 0;
            for (int64_t u = u_begin; u < u_end && ok; ++k) {
                int64_t tile;
                int c0, c1;
                seg_at(u, tile, c0, c1);
                u = tile * nchunks + c1;
                const bool has_next = u < u_end;
                // the segment's Y chunks once its tile's G is in shared memory
                ok = ok && mbar_wait(smem_u32(&g_full[k % C::NGB]), (k / C::NGB) & 1);
                tc_fence_after();
                for (int c = c0; c < c1 && ok; ++c, ++it, ++acc_it) {
                    if (C::LOOKAHEAD && c == c1 - 1 && has_next) {   // the next tile's Q, before this segment's last chunk
                        issue_q(k + 1);
                        if (!ok) break;
                    }
                    const uint32_t s = it % C::NSTAGE, ph = (it / C::NSTAGE) & 1;
                    const uint32_t ab = acc_it & 1;
                    ok = mbar_wait(smem_u32(&w_full[s]), ph) &&
                         mbar_wait(smem_u32(&acc_empty[ab]), ((acc_it >> 1) & 1) ^ 1);
                    tc_fence_after();
                    if (!ok) break;   // a wait gave up: issue nothing more
                    const uint32_t waddr = smem_u32(smem + C::OFF_W + s * C::W_STAGE_BYTES);
#pragma unroll
                    for (int kk = 0; kk < C::M / 16; ++kk) {
                        const uint64_t off = (uint64_t)(((kk / C::SPB) * (128 * C::GB) + (kk % C::SPB) * 32) >> 4);
                        const uint64_t bd = smem_desc(waddr + kk * 16 * 128, C::M * 128, 1024, kSwz128);
                        mma_bf16(tmem + ab * C::NCH, gk0 + (k % C::NGB) * TILE16 + off, bd, id_y, kk > 0);
                    }
                    mma_commit(smem_u32(&w_empty[s]));
                    mma_commit(smem_u32(&acc_full[ab]));
                }
                if (!C::LOOKAHEAD && ok && has_next) issue_q(k + 1);   // one G buffer: after this segment
            }
            mma_commit(smem_u32(&done_bar));
            mbar_wait(smem_u32(&done_bar), 0);
        }
    } else {
        // ---------------- epilogue warps (256 threads, TMEM lane quarter = warp % 4) ----------------
        const int q = warp & 3;
        const int half = (warp - 2) >> 2;   // which half of each chunk's columns this warp takes
        const int row = q * 32 + lane;
        const int et = threadIdx.x - 64;    // 0..255
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        uint32_t acc_it = 0, store_it = 0;
        bool ok = true;
        // G = phi(Q) -> bf16 -> G buffer k % NGB (K-major, NB blocks of GB-byte rows), for segment
        // k's tile whose first `valid` rows are tokens
        auto make_g = [&](uint32_t k, int valid) {
            const uint32_t ab = acc_it & 1;
            ok = ok && mbar_wait(smem_u32(&acc_full[ab]), (acc_it >> 1) & 1);
            tc_fence_after();
            if (half == 0 && ok) {   // the first four warps write G
                const bool active = row < valid;
                float g[C::M];
                tmem_ld_row<C::M>(tmem + lane_base + ab * C::NCH, g);
                tc_fence_before();
                act_fast_row<C::M>(a.act, g);
#pragma unroll
                for (int b = 0; b < C::NB; ++b) {
                    float gb[C::GB / 2];
#pragma unroll
                    for (int j = 0; j < C::GB / 2; ++j) gb[j] = active ? g[b * (C::GB / 2) + j] : 0.0f;
                    store_bf16_swz_row<C::GB / 2>(smem + C::OFF_G + (k % C::NGB) * C::TILE_BYTES + b * (128 * C::GB), row, gb);
                }
                fence_async_smem();
            }
            mbar_arrive(smem_u32(&acc_empty[ab]));
            ++acc_it;
            named_barrier(1, C::EPI);
            if (et == 0) mbar_arrive(smem_u32(&g_full[k % C::NGB]));
        };
        auto valid_of = [&](int64_t tile) -> int {
            const int64_t left = a.T - tile * 128;
            return left < 128 ? (int)left : 128;
        };
        if (u_begin < u_end) {
            int64_t tile;
            int c0, c1;
            seg_at(u_begin, tile, c0, c1);
            make_g(0, valid_of(tile));
        }
        uint32_t k = 0;
        for (int64_t u = u_begin; u < u_end && ok; ++k) {
            int64_t tile;
            int c0, c1;
            seg_at(u, tile, c0, c1);
            u = tile * nchunks + c1;
            const bool has_next = u < u_end;
            const int64_t t0 = tile * 128;
            const int valid = valid_of(tile);
            const uint8_t *bbuf = smem + C::OFF_B + (k % C::NGB) * C::TILE_BYTES;
            const float rstd = (NORM == 2 && row < valid) ? a.rstd[t0 + row] : 0.0f;   // this row's 1 / RMS
            for (int c = c0; c < c1 && ok; ++c, ++acc_it, ++store_it) {
                if (C::LOOKAHEAD && c == c1 - 1 && has_next) {   // the next tile's G (its Q was issued before this chunk)
                    int64_t nt;
                    int n0, n1;
                    seg_at(u, nt, n0, n1);
                    make_g(k + 1, valid_of(nt));
                    if (!ok) break;
                }
                const uint32_t ab = acc_it & 1;
                const uint32_t sb = store_it & 1;
                ok = mbar_wait(smem_u32(&acc_full[ab]), (acc_it >> 1) & 1);
                tc_fence_after();
                if (et == 0) bulk_wait_read<1>();  // staging buffer sb is free again
                named_barrier(1, C::EPI);
                uint8_t *stg = smem + C::OFF_STG + sb * C::STG_BYTES;
                // a warp whose 32 rows all lie past the tile's valid tokens has nothing to store
                const int gend = (q * 32 < valid) ? C::NCH : 0;
                float2 ssq = make_float2(0.0f, 0.0f);   // NORM = 1: this row's sums of squares (even, odd columns)
                // 64 columns (two TMEM loads in flight) at a time: one staging box
#pragma unroll
                for (int gh = 0; gh < C::NCH / 128; ++gh) {
                    const int g2 = half * (C::NCH / 128) + gh;   // this warp's boxes of the chunk
                    if (g2 * 64 >= gend) break;
                    float v2[2][32];
                    tmem_ld32(tmem + lane_base + ab * C::NCH + g2 * 64, v2[0]);
                    tmem_ld32(tmem + lane_base + ab * C::NCH + g2 * 64 + 32, v2[1]);
                    tmem_ld_wait();
                    tmem_regs_ready(v2[0]);
                    tmem_regs_ready(v2[1]);
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        const int g = 2 * g2 + h;   // columns [g*32, g*32+32) of the chunk
                        float (&v)[32] = v2[h];
                        // identity path: the first r columns of Y get B (only chunk 0 holds them)
                        if (g * 32 < C::R && a.merge && c == 0) {
                            const uint8_t *bblk = bbuf + ((g * 32) / (C::GB / 2)) * (128 * C::GB);
                            const uint32_t b0 = ((g * 32) % (C::GB / 2)) * 2;
#pragma unroll
                            for (int i = 0; i < 32; i += 8) {
                                if (g * 32 + i < C::R) {
                                    const uint4 u4 = *reinterpret_cast<const uint4 *>(bblk + swz_offset(row, b0 + 2 * i, C::GB));
                                    const uint32_t w[4] = {u4.x, u4.y, u4.z, u4.w};
#pragma unroll
                                    for (int e = 0; e < 4; ++e) {
                                        v[i + 2 * e] += __uint_as_float(w[e] << 16);
                                        v[i + 2 * e + 1] += __uint_as_float(w[e] & 0xFFFF0000u);
                                    }
                                }
                            }
                        }
                        uint32_t p[16];
                        if (NORM == 2) {   // gamma of these 32 columns (the same for every row)
                            const float4 *gp = reinterpret_cast<const float4 *>(a.gamma + (int64_t)c * C::NCH + g * 32);
                            const float2 r2 = make_float2(rstd, rstd);
#pragma unroll
                            for (int i = 0; i < 8; ++i) {
                                const float4 g4 = __ldg(gp + i);
#pragma unroll
                                for (int e = 0; e < 2; ++e) {
                                    const int k2 = 2 * i + e;   // the pair of columns 2 k2, 2 k2 + 1
                                    const float2 yn = __fmul2_rn(__fmul2_rn(make_float2(v[2 * k2], v[2 * k2 + 1]), r2),
                                                                 e ? make_float2(g4.z, g4.w) : make_float2(g4.x, g4.y));
                                    __nv_bfloat162 hh = __float22bfloat162_rn(yn);
                                    p[k2] = *reinterpret_cast<uint32_t *>(&hh);
                                }
                            }
                        } else {
#pragma unroll
                            for (int i = 0; i < 16; ++i) {
                                __nv_bfloat162 hh = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
                                p[i] = *reinterpret_cast<uint32_t *>(&hh);
                                if (NORM == 1) {
                                    const float2 y2 = __bfloat1622float2(hh);
                                    ssq = __ffma2_rn(y2, y2, ssq);
                                }
                            }
                        }
                        // columns [g*32, g*32+32) of the chunk: box g/2, bytes (g%2)*64 .. +64
                        uint8_t *box = stg + (g >> 1) * 16384;
                        const uint32_t b0 = (g & 1) * 64;
#pragma unroll
                        for (int i = 0; i < 4; ++i)
                            *reinterpret_cast<uint4 *>(box + swz_offset(row, b0 + 16 * i, 128)) =
                                make_uint4(p[4 * i], p[4 * i + 1], p[4 * i + 2], p[4 * i + 3]);
                    }
                }
                if (NORM == 1 && row < valid) a.ss[(int64_t)(2 * c + half) * a.T + t0 + row] = ssq.x + ssq.y;
                tc_fence_before();
                mbar_arrive(smem_u32(&acc_empty[ab]));
                fence_async_smem();
                named_barrier(1, C::EPI);
                if (et == 0) {
                    // the segment's first chunk is drained: its B rows are no longer read (the Q
                    // product and the identity path of chunk 0 are done)
                    if (c == c0) mbar_arrive(smem_u32(&b_empty[k % C::NGB]));
                    const uint32_t sbase = smem_u32(stg);
                    for (int b = 0; b < C::NCH / 64; ++b) {
                        const int x = c * C::NCH + 64 * b;
                        if (valid == 128) {
                            tma_store_2d_hint(&tm_y128, x, (int32_t)t0, sbase + b * 16384, l2_evict_first());
                        } else {
                            for (int rg = 0; rg * 16 < valid; ++rg)
                                tma_store_2d_hint(&tm_y16, x, (int32_t)(t0 + 16 * rg), sbase + b * 16384 + rg * 2048, l2_evict_first());
                        }
                    }
                    bulk_commit();
                }
            }
            if (!C::LOOKAHEAD && ok && has_next) {   // one G buffer: the next tile's G after this segment
                int64_t nt;
                int n0, n1;
                seg_at(u, nt, n0, n1);
                make_g(k + 1, valid_of(nt));
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
