// tc_enc_fwd.cuh -- send side of the boundary on tensor cores (Sec. 3.2 encoder, Eq. Pid
// truncating identity path):  P = F . We1 (saved, fp32),  B = X[:, :r] + phi(P) . We2.
//
// Persistent CTAs over contiguous 16-token-aligned token ranges, tiles of up to 128 tokens.
//   producer warp : for each tile, d in chunks of 64 columns: F tile chunk (128 x 64, K-major,
//                   128B swizzle; 16-row boxes for a partial tile) + We1 rows (64 x m, MN-major)
//   MMA warp      : P (128 x m fp32 in TMEM, double-buffered per tile) += F_chunk . We1_chunk
//   epilogue warps: TMEM -> registers (one token per thread), store P, A = phi(P),
//                   E = A . We2 (fp32 on CUDA cores, We2 in shared memory), B = X[:, :r] + E
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
    static constexpr int NSTAGE = M_ <= 32 ? 8 : (M_ == 64 ? 6 : 5);
    static constexpr uint32_t WE2_BYTES = M_ * R * 2;
    static constexpr uint32_t OFF_STAGE = 0;
    static constexpr uint32_t OFF_WE2 = NSTAGE * STAGE_BYTES;
    static constexpr uint32_t SMEM_BYTES = OFF_WE2 + WE2_BYTES + 1024;
    static constexpr uint32_t ACC_STRIDE = M_ < 32 ? 32 : M_;          // TMEM columns per accumulator
    static constexpr uint32_t TMEM_COLS = 2 * ACC_STRIDE;
    static constexpr int THREADS = 192;
};

struct EncFwdArgs {
    const __nv_bfloat16 *X;    // T x d (first r columns read)
    const __nv_bfloat16 *We2;  // m x r
    __nv_bfloat16 *B;          // T x r
    float *P;                  // T x m or null
    int64_t T, d;
    int act;
};

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
    __shared__ uint64_t full[C::NSTAGE], empty[C::NSTAGE];
    __shared__ uint64_t acc_full[2], acc_empty[2], done_bar;
    __shared__ uint32_t tmem_base_sh;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nk = (int)(a.d / 64);
    int64_t start, end;
    token_range(a.T, blockIdx.x, gridDim.x, start, end);

    if (threadIdx.x == 0) {
        for (int s = 0; s < C::NSTAGE; ++s) {
            mbar_init(smem_u32(&full[s]), 1);
            mbar_init(smem_u32(&empty[s]), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(smem_u32(&acc_full[i]), 1);
            mbar_init(smem_u32(&acc_empty[i]), 128);
        }
        mbar_init(smem_u32(&done_bar), 1);
        fence_mbar_init();
    }
    if (warp == 1) tmem_alloc(smem_u32(&tmem_base_sh), C::TMEM_COLS);
    if (warp >= 2) {  // We2 (m x r bf16) into shared memory, once
        const uint4 *src = reinterpret_cast<const uint4 *>(a.We2);
        uint4 *dst = reinterpret_cast<uint4 *>(smem + C::OFF_WE2);
        for (int i = threadIdx.x - 64; i < (int)(C::WE2_BYTES / 16); i += 128) dst[i] = src[i];
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_base_sh;

    if (warp == 0) {
        // ---------------- producer ----------------
        if (elect_one()) {
            tma_prefetch_desc(&tm_f128);
            tma_prefetch_desc(&tm_f16);
            tma_prefetch_desc(&tm_we1);
            uint32_t it = 0;
            bool ok = true;
            for (int64_t t0 = start; t0 < end && ok; t0 += 128) {
                const int valid = (int)((end - t0) < 128 ? (end - t0) : 128);
                const int nbox16 = (valid + 15) / 16;
                const uint32_t fbytes = valid == 128 ? C::F_BYTES : (uint32_t)nbox16 * 2048u;
                for (int kc = 0; kc < nk; ++kc) {
                    const uint32_t s = it % C::NSTAGE, ph = (it / C::NSTAGE) & 1;
                    if (!mbar_wait(smem_u32(&empty[s]), ph ^ 1)) {
                        ok = false;
                        break;
                    }
                    const uint32_t fdst = smem_u32(smem + C::OFF_STAGE + s * C::STAGE_BYTES);
                    const uint32_t wdst = fdst + C::F_BYTES;
                    const uint32_t bar = smem_u32(&full[s]);
                    mbar_expect_tx(bar, fbytes + C::W_BYTES);
                    if (valid == 128) {
                        tma_load_2d(fdst, &tm_f128, kc * 64, (int32_t)t0, bar);
                    } else {
                        for (int rg = 0; rg < nbox16; ++rg)
                            tma_load_2d(fdst + rg * 2048, &tm_f16, kc * 64, (int32_t)(t0 + 16 * rg), bar);
                    }
                    for (int wb = 0; wb < C::WBOXES; ++wb)
                        tma_load_2d(wdst + wb * 64 * C::WSW, &tm_we1, wb * 64, kc * 64, bar);
                    ++it;
                }
            }
            const uint32_t n = it < (uint32_t)C::NSTAGE ? it : (uint32_t)C::NSTAGE;
            for (uint32_t k = 0; k < n; ++k) {
                const uint32_t j = it - 1 - k;
                mbar_wait(smem_u32(&full[j % C::NSTAGE]), (j / C::NSTAGE) & 1);
            }
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if (elect_one()) {
            constexpr Swz wswz = C::WSW == 128 ? kSwz128 : C::WSW == 64 ? kSwz64 : kSwz32;
            constexpr uint32_t idesc = idesc_bf16(128, C::M, false, true);
            uint32_t it = 0, tile_i = 0;
            bool ok = true;
            for (int64_t t0 = start; t0 < end && ok; t0 += 128, ++tile_i) {
                const uint32_t ab = tile_i & 1;
                ok = mbar_wait(smem_u32(&acc_empty[ab]), ((tile_i >> 1) & 1) ^ 1);
                tc_fence_after();
                for (int kc = 0; kc < nk && ok; ++kc, ++it) {
                    const uint32_t s = it % C::NSTAGE, ph = (it / C::NSTAGE) & 1;
                    ok = mbar_wait(smem_u32(&full[s]), ph);
                    tc_fence_after();
                    const uint32_t faddr = smem_u32(smem + C::OFF_STAGE + s * C::STAGE_BYTES);
                    const uint32_t waddr = faddr + C::F_BYTES;
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const uint64_t ad = smem_desc(faddr + k * 32, 16, 1024, kSwz128);
                        const uint64_t bd = smem_desc(waddr + k * 16 * C::WSW, 64 * C::WSW, 8 * C::WSW, wswz);
                        mma_bf16(tmem + ab * C::ACC_STRIDE, ad, bd, idesc, (kc | k) != 0);
                    }
                    mma_commit(smem_u32(&empty[s]));
                }
                mma_commit(smem_u32(&acc_full[ab]));
            }
            mma_commit(smem_u32(&done_bar));
            mbar_wait(smem_u32(&done_bar), 0);
        }
    } else {
        // ---------------- epilogue: one token per thread ----------------
        const int q = warp & 3;
        const int row = q * 32 + lane;
        const __nv_bfloat16 *we2 = reinterpret_cast<const __nv_bfloat16 *>(smem + C::OFF_WE2);
        uint32_t tile_i = 0;
        bool ok = true;
        for (int64_t t0 = start; t0 < end && ok; t0 += 128, ++tile_i) {
            const int valid = (int)((end - t0) < 128 ? (end - t0) : 128);
            const uint32_t ab = tile_i & 1;
            ok = mbar_wait(smem_u32(&acc_full[ab]), (tile_i >> 1) & 1);
            tc_fence_after();
            float p[C::M];
#pragma unroll
            for (int j = 0; j < C::M; j += 16) {
                float v[16];
                tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + ab * C::ACC_STRIDE + j, v);
                tmem_ld_wait();
#pragma unroll
                for (int i = 0; i < 16; ++i) p[j + i] = v[i];
            }
            tc_fence_before();
            mbar_arrive(smem_u32(&acc_empty[ab]));
            if (row < valid) {  // (with a.B == null only P is wanted: P = F . We1 for the backward)
                const int64_t tok = t0 + row;
                if (a.P) {
                    float4 *dst = reinterpret_cast<float4 *>(a.P + tok * C::M);
#pragma unroll
                    for (int j = 0; j < C::M / 4; ++j)
                        dst[j] = make_float4(p[4 * j], p[4 * j + 1], p[4 * j + 2], p[4 * j + 3]);
                }
                act_row<C::M>(a.act, p);
                const uint4 *xs = reinterpret_cast<const uint4 *>(a.X + tok * a.d);
                uint4 *bd = reinterpret_cast<uint4 *>(a.B + tok * C::R);
#pragma unroll
                for (int jb = 0; jb < C::R; jb += 8) {
                    if (a.B == nullptr) break;
                    // E[jb .. jb+8) = sum_j A[j] We2[j][jb .. jb+8), fp32
                    float e[8];
#pragma unroll
                    for (int i = 0; i < 8; ++i) e[i] = 0.0f;
#pragma unroll
                    for (int j = 0; j < C::M; ++j) {
                        const uint4 w = *reinterpret_cast<const uint4 *>(we2 + j * C::R + jb);
                        const uint32_t wv[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            e[2 * i] = fmaf(p[j], __uint_as_float(wv[i] << 16), e[2 * i]);
                            e[2 * i + 1] = fmaf(p[j], __uint_as_float(wv[i] & 0xFFFF0000u), e[2 * i + 1]);
                        }
                    }
                    const uint4 x = xs[jb / 8];
                    const uint32_t xv[4] = {x.x, x.y, x.z, x.w};
                    uint32_t o[4];
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const float b0 = __uint_as_float(xv[i] << 16) + e[2 * i];
                        const float b1 = __uint_as_float(xv[i] & 0xFFFF0000u) + e[2 * i + 1];
                        __nv_bfloat162 h = __floats2bfloat162_rn(b0, b1);
                        o[i] = *reinterpret_cast<uint32_t *>(&h);
                    }
                    bd[jb / 8] = make_uint4(o[0], o[1], o[2], o[3]);
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
}

}  // namespace tc
}  // namespace resbm
