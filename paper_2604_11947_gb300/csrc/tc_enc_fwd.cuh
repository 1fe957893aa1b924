// tc_enc_fwd.cuh -- send side of the boundary on tensor cores (Sec. 3.2 encoder, Eq. Pid
// truncating identity path):  P = F . We1 (saved, fp32),  B = X[:, :r] + phi(P) . We2.
//
// Persistent CTAs in pairs (clusters of 2; single CTAs for m = 128): each pair owns a
// contiguous run of whole 128-token tiles (balanced over the pairs) and splits it evenly in
// 64-column chunks, so at most one tile is shared: rank 1 takes the shared tile's last chunks
// first and pushes its partial P (128 x m fp32) into rank 0's shared memory (st.async, counted
// on rank 0's barrier), and rank 0 takes the tile's first chunks last, adds the two partials in
// rank order (P = P_rank0 + P_rank1, a fixed order) and finishes the tile. A CTA's pipeline is
// paced by its stages, not by bytes, so at T = 65536 the pairs make at most 3.5 tile passes
// instead of 4 (the tensor's last tile may be partial).
//   producer warp : for each tile, d in chunks of 64 columns: F tile chunk (128 x 64, K-major,
//                   128B swizzle; 16-row boxes for a partial tile) + We1 rows (64 x m, MN-major),
//                   two consecutive chunks per ring stage for m <= 32
//   MMA warp      : P (128 x m fp32 in TMEM, double-buffered per tile) += F_chunk . We1_chunk
//   epilogue warps: TMEM -> registers (one token per thread), store P, A = phi(P) as a bf16
//                   hi + lo pair in shared memory; the MMA warp then computes E = A . We2 into
//                   TMEM (polled between the next tile's stages); B = X[:, :r] + E
// HBM traffic per token: read F (2d), X[:, :r] (2r); write B (2r), P (4m).
#pragma once

#include "common.cuh"
#include "tc_common.cuh"

namespace resbm {
namespace tc {

template <int M_> struct EncFwdCfg {
    static constexpr int M = M_;
    static constexpr int R = M_;
    static constexpr uint32_t WSW = M_ >= 64 ? 128 : M_ * 2;          // We1 box row bytes (swizzle)
    static constexpr int WBOXES = M_ >= 64 ? M_ / 64 : 1;             // We1 boxes per chunk
    static constexpr uint32_t F_BYTES = 128 * 128;                      // 128 rows x 64 bf16
    static constexpr uint32_t W_BYTES = 64 * M_ * 2;                    // 64 rows x m bf16
    static constexpr uint32_t STAGE_BYTES = F_BYTES + W_BYTES;
    static constexpr int NSTAGE = M_ <= 32 ? 8 : (M_ == 64 ? 6 : 3);   // chunk slots
    // chunks per ring stage (one barrier, one wait per stage): two consecutive 64-column chunks
    // of a tile share a stage for m <= 32 (a tile's odd last chunk fills half a stage); per CTA
    // the stream is paced by stages in flight, and 32 KB of F per stage streams faster than 16
    static constexpr int SUB = M_ <= 32 ? 2 : 1;
    static constexpr int NST = NSTAGE / SUB;                            // ring stages
    static constexpr uint32_t GB = M_ * 2 < 128 ? M_ * 2 : 128;        // row bytes (= swizzle) of an A block
    static constexpr int NB = M_ * 2 / GB;                              // blocks across the m columns
    static constexpr int SPB = GB / 32;                                 // 16-element K steps per block
    static constexpr uint32_t A_TILE = 128 * M_ * 2;                    // 128 tokens x m bf16
    static constexpr uint32_t WE2T_BYTES = R * M_ * 2;
    static constexpr uint32_t OFF_STAGE = 0;
    static constexpr uint32_t OFF_A = NSTAGE * STAGE_BYTES;             // A = phi(P): hi tile, then lo tile
    static constexpr uint32_t OFF_WE2T = OFF_A + 2 * A_TILE;            // We2^T [r][m], K-major
    static constexpr bool SPLIT = M_ <= 64;                              // tiles shared within a pair
    static constexpr uint32_t OFF_RX = OFF_WE2T + WE2T_BYTES;           // the peer's partial P [128][m] fp32
    static constexpr uint32_t SMEM_BYTES = OFF_RX + (SPLIT ? 128 * M_ * 4 : 0) + 1024;
    static_assert(SMEM_BYTES <= 232448 - 512, "shared memory budget");
    static constexpr uint32_t ACC_STRIDE = M_ < 32 ? 32 : M_;          // TMEM columns per accumulator
    static constexpr uint32_t TM_E = 2 * ACC_STRIDE;                    // E = A . We2 (r columns)
    static constexpr uint32_t TMEM_NEED = TM_E + ACC_STRIDE;
    static constexpr uint32_t TMEM_COLS = TMEM_NEED <= 128 ? 128 : TMEM_NEED <= 256 ? 256 : 512;
    static constexpr int THREADS = 192;
};

struct EncFwdArgs {
    const __nv_bfloat16 *X;    // T x d (first r columns read)
    const __nv_bfloat16 *We2;  // m x r
    __nv_bfloat16 *B;          // T x r, or null: P = F . We1 only (for the backward)
    float *P;                  // T x m or null
    int64_t T, d;
    int act;
};

// Work of one CTA: tiles [t_begin, t_end), the first from 64-column chunk kc_first, the last up
// to chunk kc_last (exclusive). A pair (cl = 2) splits its tiles' chunks evenly: rank 0 takes
// the first half (its last tile possibly partial: recv_last), rank 1 the second (its first tile
// possibly partial: send_first).
struct EncFwdWork {
    int64_t t_begin, t_end;
    int kc_first, kc_last;
    bool send_first, recv_last;
};
__device__ __forceinline__ EncFwdWork enc_fwd_work(int64_t T, int nk, uint32_t cl, uint32_t rank, uint32_t cid,
                                                   uint32_t ncl)
{
    const int64_t U = (T + 127) / 128;
    const int64_t a = U * cid / ncl, b = U * (cid + 1) / ncl;
    EncFwdWork w{a, b, 0, nk, false, false};
    if (cl < 2) return w;
    const int64_t L = (b - a) * nk, half = L / 2;
    if (rank == 0) {
        if (half == 0) {
            w.t_end = a;   // nothing
        } else {
            w.t_end = a + (half - 1) / nk + 1;
            w.kc_last = (int)((half - 1) % nk) + 1;
            w.recv_last = half % nk != 0;
        }
    } else {
        w.t_begin = a + half / nk;
        w.kc_first = (int)(half % nk);
        w.send_first = half % nk != 0;
    }
    return w;
}

template <int M_>
__global__ void __launch_bounds__(192, 1)
    k_enc_fwd(const __grid_constant__ CUtensorMap tm_f128, const __grid_constant__ CUtensorMap tm_f16,
              const __grid_constant__ CUtensorMap tm_we1, const EncFwdArgs a)
{
    using C = EncFwdCfg<M_>;
    griddep_wait();               // the previous kernel of the stream has completed
    griddep_launch_dependents();  // the next one may be scheduled on SMs as they free up
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    __shared__ uint64_t full[C::NST], empty[C::NST];
    __shared__ uint64_t acc_full[2], acc_empty[2], a_full, e_full, done_bar, rx_full;
    __shared__ uint32_t tmem_base_sh;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nk = (int)(a.d / 64);
    const bool want_b = a.B != nullptr;
    const uint32_t cl = C::SPLIT ? cluster_size() : 1u;
    const EncFwdWork wk = enc_fwd_work(a.T, nk, cl, C::SPLIT ? cluster_rank() : 0u, cluster_index(), gridDim.x / cl);
    const int ntiles = (int)(wk.t_end - wk.t_begin);
    // the tiles that need E = A . We2 (all but a tile whose partial P goes to the peer)
    const int e_tiles = ntiles - (wk.send_first ? 1 : 0);
    auto chunks_of = [&](int ti, int &kc0, int &kc1) {
        kc0 = ti == 0 ? wk.kc_first : 0;
        kc1 = ti == ntiles - 1 ? wk.kc_last : nk;
    };
    auto valid_of = [&](int ti) -> int {
        const int64_t left = a.T - (wk.t_begin + ti) * 128;
        return left < 128 ? (int)left : 128;
    };

    if (threadIdx.x == 0) {
        for (int s = 0; s < C::NST; ++s) {
            mbar_init(smem_u32(&full[s]), 1);
            mbar_init(smem_u32(&empty[s]), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(smem_u32(&acc_full[i]), 1);
            mbar_init(smem_u32(&acc_empty[i]), 128);
        }
        mbar_init(smem_u32(&a_full), 1);
        mbar_init(smem_u32(&e_full), 1);
        mbar_init(smem_u32(&done_bar), 1);
        mbar_init(smem_u32(&rx_full), 1);
        fence_mbar_init();
        // the peer's partial P of the shared tile: 128 rows of m fp32
        if (wk.recv_last) mbar_expect_tx(smem_u32(&rx_full), 128 * C::M * 4);
    }
    if (warp == 1) tmem_alloc(smem_u32(&tmem_base_sh), C::TMEM_COLS);
    if (warp >= 2 && want_b) {  // We2^T (r x m) as a swizzled K-major operand: NB blocks of GB-byte rows
        for (int e = threadIdx.x - 64; e < C::M * C::R; e += 128) {
            const int k = e / C::R, n = e % C::R;   // We2[k][n]
            const int kb = k / (C::GB / 2), kk = k % (C::GB / 2);
            *reinterpret_cast<__nv_bfloat16 *>(smem + C::OFF_WE2T + kb * (C::R * C::GB) + swz_offset(n, 2 * kk, C::GB)) =
                a.We2[e];
        }
        fence_async_smem();
    }
    tc_fence_before();
    __syncthreads();
    if (C::SPLIT && cl > 1) cluster_sync();   // the peer's barrier is armed before anything is pushed
    tc_fence_after();
    const uint32_t tmem = tmem_base_sh;

    if (warp == 0) {
        // ---------------- producer ----------------
        if (elect_one()) {
            const uint64_t stream_pol = l2_evict_first();   // read once
            tma_prefetch_desc(&tm_f128);
            tma_prefetch_desc(&tm_f16);
            tma_prefetch_desc(&tm_we1);
            uint32_t it = 0;
            bool ok = true;
            for (int ti = 0; ti < ntiles && ok; ++ti) {
                const int64_t t0 = (wk.t_begin + ti) * 128;
                const int valid = valid_of(ti);
                const int nbox16 = (valid + 15) / 16;
                const uint32_t fbytes = valid == 128 ? C::F_BYTES : (uint32_t)nbox16 * 2048u;
                int kc0, kc1;
                chunks_of(ti, kc0, kc1);
                for (int kc = kc0; kc < kc1; kc += C::SUB) {
                    const int nsub = kc1 - kc < C::SUB ? kc1 - kc : C::SUB;   // chunks in this stage
                    const uint32_t s = it % C::NST, ph = (it / C::NST) & 1;
                    if (!mbar_wait(smem_u32(&empty[s]), ph ^ 1)) {
                        ok = false;
                        break;
                    }
                    const uint32_t bar = smem_u32(&full[s]);
                    mbar_expect_tx(bar, (uint32_t)nsub * (fbytes + C::W_BYTES));
                    for (int j = 0; j < nsub; ++j) {
                        const uint32_t fdst = smem_u32(smem + C::OFF_STAGE + (s * C::SUB + j) * C::STAGE_BYTES);
                        const uint32_t wdst = fdst + C::F_BYTES;
                        if (valid == 128) {
                            tma_load_2d_hint(fdst, &tm_f128, (kc + j) * 64, (int32_t)t0, bar, stream_pol);
                        } else {
                            for (int rg = 0; rg < nbox16; ++rg)
                                tma_load_2d_hint(fdst + rg * 2048, &tm_f16, (kc + j) * 64, (int32_t)(t0 + 16 * rg), bar,
                                                 stream_pol);
                        }
                        for (int wb = 0; wb < C::WBOXES; ++wb)
                            tma_load_2d(wdst + wb * 64 * C::WSW, &tm_we1, wb * 64, (kc + j) * 64, bar);
                    }
                    ++it;
                }
            }
            const uint32_t n = it < (uint32_t)C::NST ? it : (uint32_t)C::NST;
            for (uint32_t k = 0; k < n; ++k) {
                const uint32_t j = it - 1 - k;
                mbar_wait(smem_u32(&full[j % C::NST]), (j / C::NST) & 1);
            }
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if (elect_one()) {
            constexpr Swz wswz = C::WSW == 128 ? kSwz128 : C::WSW == 64 ? kSwz64 : kSwz32;
            constexpr Swz gsw = swz_for(C::GB);
            constexpr uint32_t idesc = idesc_bf16(128, C::M, false, true);
            constexpr uint32_t id_e = idesc_bf16(128, C::R, false, false);   // A (K-major) . We2^T rows (K-major)
            const uint64_t ak0 = smem_desc(smem_u32(smem + C::OFF_A), 16, 8 * C::GB, gsw);
            const uint64_t wt0 = smem_desc(smem_u32(smem + C::OFF_WE2T), 16, 8 * C::GB, gsw);
            constexpr uint64_t LO16 = C::A_TILE >> 4;
            // E = (A_hi + A_lo) . We2 of the tile whose A the epilogue has published
            uint32_t e_issued = 0;
            auto issue_e = [&]() {
#pragma unroll
                for (int k = 0; k < C::M / 16; ++k) {
                    const uint64_t off = (uint64_t)(((k / C::SPB) * (128 * C::GB) + (k % C::SPB) * 32) >> 4);
                    const uint64_t woff = (uint64_t)(((k / C::SPB) * (C::R * C::GB) + (k % C::SPB) * 32) >> 4);
                    mma_bf16(tmem + C::TM_E, ak0 + off, wt0 + woff, id_e, k > 0);
                    mma_bf16(tmem + C::TM_E, ak0 + LO16 + off, wt0 + woff, id_e, true);
                }
                mma_commit(smem_u32(&e_full));
                ++e_issued;
            };
            uint32_t it = 0, e_ready = 0;   // e_ready: E tiles whose P product has been committed
            // Wait for (bar, parity) while issuing, in the meantime, the E product of an earlier
            // tile as soon as the epilogue publishes its A: the epilogue waits for that E before
            // it frees the accumulators this thread may be waiting for, so no wait may block it.
            auto wait_serving_e = [&](uint32_t bar, uint32_t parity) -> bool {
                const unsigned long long t_start = globaltimer();
                for (uint32_t i = 0;; ++i) {
                    if (want_b && e_issued < e_ready && mbar_test_wait(smem_u32(&a_full), e_issued & 1)) {
                        tc_fence_after();
                        issue_e();
                    }
                    if (mbar_try_wait(bar, parity)) return true;
                    if ((i & 255u) == 0 && globaltimer() - t_start > kWaitNs) {
                        flag_error(kErrWaitTimeout);
                        return false;
                    }
                }
            };
            bool ok = true;
            for (int ti = 0; ti < ntiles && ok; ++ti) {
                const uint32_t ab = ti & 1;
                ok = wait_serving_e(smem_u32(&acc_empty[ab]), ((ti >> 1) & 1) ^ 1);
                tc_fence_after();
                if (!ok) break;
                int kc0, kc1;
                chunks_of(ti, kc0, kc1);
                for (int kc = kc0; kc < kc1 && ok; kc += C::SUB, ++it) {
                    const int nsub = kc1 - kc < C::SUB ? kc1 - kc : C::SUB;
                    const uint32_t s = it % C::NST, ph = (it / C::NST) & 1;
                    ok = wait_serving_e(smem_u32(&full[s]), ph);
                    tc_fence_after();
                    if (!ok) break;   // a wait gave up: issue nothing more
                    for (int j = 0; j < nsub; ++j) {
                        const uint32_t faddr = smem_u32(smem + C::OFF_STAGE + (s * C::SUB + j) * C::STAGE_BYTES);
                        const uint32_t waddr = faddr + C::F_BYTES;
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const uint64_t ad = smem_desc(faddr + k * 32, 16, 1024, kSwz128);
                            const uint64_t bd = smem_desc(waddr + k * 16 * C::WSW, 64 * C::WSW, 8 * C::WSW, wswz);
                            mma_bf16(tmem + ab * C::ACC_STRIDE, ad, bd, idesc, kc + j != kc0 || k != 0);
                        }
                    }
                    mma_commit(smem_u32(&empty[s]));
                }
                mma_commit(smem_u32(&acc_full[ab]));
                if (!(ti == 0 && wk.send_first)) ++e_ready;
            }
            // the E products not issued inside the stream (at least the last tile's)
            while (ok && want_b && e_issued < (uint32_t)e_tiles) {
                ok = mbar_wait(smem_u32(&a_full), e_issued & 1);
                tc_fence_after();
                if (ok) issue_e();
            }
            mma_commit(smem_u32(&done_bar));
            mbar_wait(smem_u32(&done_bar), 0);
        }
    } else {
        // ---------------- epilogue: one token per thread ----------------
        const int q = warp & 3;
        const int row = q * 32 + lane;
        const int et = threadIdx.x - 64;
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        uint32_t ei = 0;   // E tiles so far
        bool ok = true;
        for (int ti = 0; ti < ntiles && ok; ++ti) {
            const int64_t t0 = (wk.t_begin + ti) * 128;
            const int valid = valid_of(ti);
            const bool active = row < valid;
            const int64_t tok = t0 + row;
            const uint32_t ab = ti & 1;
            ok = mbar_wait(smem_u32(&acc_full[ab]), (ti >> 1) & 1);
            tc_fence_after();
            float p[C::M];
            tmem_ld_row<C::M>(tmem + lane_base + ab * C::ACC_STRIDE, p);
            tc_fence_before();
            mbar_arrive(smem_u32(&acc_empty[ab]));
            if (C::SPLIT) {
                constexpr int V4 = C::M / 4, SW = V4 < 8 ? V4 - 1 : 7;   // float4 per row, swizzle mask
                const uint32_t rx = smem_u32(smem + C::OFF_RX) + (uint32_t)row * (C::M * 4);
                if (ti == 0 && wk.send_first) {
                    // this tile's last chunks were ours: the partial P goes to rank 0, which adds it
                    const uint32_t dst = map_shared(rx, 0), bar = map_shared(smem_u32(&rx_full), 0);
#pragma unroll
                    for (int e = 0; e < V4; ++e)
                        st_async_f4(dst + 16u * (uint32_t)(e ^ (row & SW)),
                                    make_float4(p[4 * e], p[4 * e + 1], p[4 * e + 2], p[4 * e + 3]), bar);
                    continue;
                }
                if (ti == ntiles - 1 && wk.recv_last) {
                    // P = our partial (the tile's first chunks) + rank 1's (its last chunks)
                    ok = mbar_wait(smem_u32(&rx_full), 0);
#pragma unroll
                    for (int e = 0; e < V4; ++e) {
                        float4 x;
                        asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
                                     : "=f"(x.x), "=f"(x.y), "=f"(x.z), "=f"(x.w)
                                     : "r"(rx + 16u * (uint32_t)(e ^ (row & SW)))
                                     : "memory");
                        p[4 * e] = p[4 * e] + x.x;
                        p[4 * e + 1] = p[4 * e + 1] + x.y;
                        p[4 * e + 2] = p[4 * e + 2] + x.z;
                        p[4 * e + 3] = p[4 * e + 3] + x.w;
                    }
                }
            }
            if (active && a.P) {
                float4 *dst = reinterpret_cast<float4 *>(a.P + tok * C::M);
#pragma unroll
                for (int j = 0; j < C::M / 4; ++j)
                    dst[j] = make_float4(p[4 * j], p[4 * j + 1], p[4 * j + 2], p[4 * j + 3]);
            }
            if (!want_b) continue;   // P only
            // this token's X[:, :r], fetched now and used after E
            float xv[C::R];
#pragma unroll
            for (int j = 0; j < C::R; ++j) xv[j] = 0.0f;
            if (active) load_bf16_row<C::R>(a.X + tok * a.d, xv);
            // A = phi(P) as bf16 hi + lo (the E product then sees A to about 16 significant bits)
            act_row<C::M>(a.act, p);
#pragma unroll
            for (int b = 0; b < C::NB; ++b) {
                float hi[C::GB / 2], lo[C::GB / 2];
#pragma unroll
                for (int j = 0; j < C::GB / 2; ++j) {
                    const float x = active ? p[b * (C::GB / 2) + j] : 0.0f;
                    hi[j] = __bfloat162float(__float2bfloat16_rn(x));
                    lo[j] = x - hi[j];
                }
                store_bf16_swz_row<C::GB / 2>(smem + C::OFF_A + b * (128 * C::GB), row, hi);
                store_bf16_swz_row<C::GB / 2>(smem + C::OFF_A + C::A_TILE + b * (128 * C::GB), row, lo);
            }
            fence_async_smem();
            named_barrier(1, 128);
            if (et == 0) mbar_arrive(smem_u32(&a_full));
            // B = X[:, :r] + E
            ok = mbar_wait(smem_u32(&e_full), ei & 1);
            ++ei;
            tc_fence_after();
            float e[C::R];
            tmem_ld_row<C::R>(tmem + lane_base + C::TM_E, e);
            tc_fence_before();
            if (active) {
                uint4 *bd = reinterpret_cast<uint4 *>(a.B + tok * C::R);
#pragma unroll
                for (int v8 = 0; v8 < C::R / 8; ++v8) {
                    uint32_t o[4];
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        __nv_bfloat162 h = __floats2bfloat162_rn(xv[8 * v8 + 2 * i] + e[8 * v8 + 2 * i],
                                                                 xv[8 * v8 + 2 * i + 1] + e[8 * v8 + 2 * i + 1]);
                        o[i] = *reinterpret_cast<uint32_t *>(&h);
                    }
                    bd[v8] = make_uint4(o[0], o[1], o[2], o[3]);
                }
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, C::TMEM_COLS);
    }
    if (C::SPLIT && cl > 1) cluster_sync();   // no peer addresses this CTA's shared memory any more
}

}  // namespace tc
}  // namespace resbm
