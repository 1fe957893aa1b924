// tc_gemm.cuh -- a persistent tcgen05 GEMM with the boundary's epilogues fused in, for the
// widths the fused boundary kernels do not take (m = r = 512, the r = 128 backward, m != r):
// there the two linear layers of Sec. 3.2's encoder and decoder, and their gradients, become a
// chain of products C = A . B (bf16 operands, fp32 accumulation in TMEM), each with the
// element-wise step that follows it in the chain (phi, phi', the identity-path merge of Eq. Pid,
// the residual-gradient update) applied to the accumulator before it leaves the chip.
//
//   C[M x N] = sum over k of A[m][k] . B[k][n]
//   A: K-major (stored M x K row-major) or MN-major (stored K x M row-major, i.e. A^T in memory)
//   B: K-major (stored N x K row-major) or MN-major (stored K x N row-major)
//
// Work units are (128-row block, BN-column block, K split); unit u runs on CTA u mod grid
// (n fastest, then m, then the split: CTAs running at the same time share their A block and,
// across a wave, their B rows in L2). Per CTA:
//   producer warp  : TMA loads of 64-deep K slices of A (128 x 64) and B (BN x 64), 128-byte
//                    swizzle, into a ring of NST stages
//   MMA warp       : four 128 x BN x 16 tcgen05.mma per stage into one of two TMEM accumulators
//                    (double-buffered: the next unit's products overlap this unit's epilogue)
//   With ALO the A operand is a bf16 pair hi + lo (hi = a value rounded to bf16, lo = the
//   rounded remainder, two matrices of the same shape): each stage holds both A tiles and the
//   MMA warp issues hi . B and lo . B into the same accumulator, so the product sees A to about
//   16 significant bits (used where the result crosses the boundary, B and dB, and for the
//   decoder's dWd2 = G^T . dY, a long sum over tokens whose terms cancel for real gradients).
//   epilogue warps : eight warps, two per TMEM lane quarter splitting the columns: TMEM ->
//                    registers (one output row per thread, 32 columns at a time) -> the
//                    epilogue's element-wise step -> global memory
// Out-of-range rows, columns and K are read as zeros by TMA and never written, so any M, N, K
// with 16-byte row pitches work. Each output element is summed by one CTA in K order (a split-K
// launch writes per-split fp32 slots that a second kernel adds in slot order), so results are
// bitwise reproducible.
#pragma once

#include "common.cuh"
#include "tc_common.cuh"

namespace resbm {
namespace tc {

// tma_load_2d multicast to the CTAs of the cluster in cta_mask: the box lands at the same
// shared-memory offset in each of them and completes its bytes on the mbarrier at the same
// offset in each (this GPU's own memory only).
__device__ __forceinline__ void tma_load_2d_mc(uint32_t dst, const CUtensorMap *m, int32_t x, int32_t y, uint32_t bar,
                                               uint16_t cta_mask)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.multicast::cluster"
        " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(m)), "r"(x), "r"(y), "r"(bar), "h"(cta_mask)
        : "memory");
}

// mma_commit arriving on the mbarrier at the same offset in every CTA of the cluster in cta_mask.
__device__ __forceinline__ void mma_commit_mc(uint32_t bar, uint16_t cta_mask)
{
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(bar),
        "h"(cta_mask)
        : "memory");
}

// The element-wise step after the product (acc = the fp32 accumulator of one output element at
// row `row`, column `col`; phi and phi' as in common.cuh; every bf16 result rounded once to
// nearest even).
// `lo` (if set) receives the rounded remainder of the bf16 activation result named below, so that
// a later product can use it as a hi + lo pair.
enum GemmEpMode : int {
    GEP_F32 = 0,   // out f32 = acc (with split-K: slot ks at out + ks * split_stride)
    GEP_BF16,      // out bf16 = acc
    GEP_P_A,       // out f32 = acc (if out), out2 bf16 = phi(acc) (lo: its remainder)  (P, A)
    GEP_ADD_AUX,   // out bf16 = acc + aux[row][col] for col < aux_cols, acc elsewhere  (B, Y, dB)
    GEP_ACT,       // out bf16 = phi(acc) (lo: its remainder), out2 f32 = acc if out2   (G, Q)
    GEP_DACT,      // out bf16 = acc * phi'(aux f32) (lo: its remainder), out2 bf16 = phi(aux) if
                   // out2                                                              (dQ; dP, A)
    GEP_DF,        // out bf16 = acc; rmw[row][col] += aux[row][col] for col < aux_cols (dF; dX += dB)
    GEP_AXPBY,     // out bf16 = alpha * acc + beta * aux[row][col] (aux bf16; the Newton-Schulz steps)
};

struct GemmEp {
    int mode, act;
    void *out;           // ldo elements per row
    int64_t ldo;
    void *out2;          // ldo2 elements per row
    int64_t ldo2;
    const void *aux;     // bf16 (ADD_AUX, DF) or f32 (DACT); lda elements per row
    int64_t lda, aux_cols;
    __nv_bfloat16 *rmw;  // DF: ldr elements per row
    int64_t ldr;
    int64_t split_stride;
    __nv_bfloat16 *lo;   // P_A, ACT, DACT: the remainder of the bf16 activation result (same pitch)
    float alpha, beta;   // AXPBY
    // ENCP launches (the encoder fused into the FFN down-projection): F = acc rounded to bf16
    // (stored at out if set), and the partial P_slice = F_tile . We1[cols of the tile] summed over
    // a thread's BN / 2 columns, written to slot (nb * 2 + half) of pslots (slots T x pm fp32,
    // slot_stride apart)
    const __nv_bfloat16 *we1;   // d x pm
    float *pslots;
    int64_t slot_stride;
    int pm;
};

// P partial of one row over 32 columns: pacc[j] += sum over c of f[c] * We1[col + c][j], j < m
// (m a multiple of 8, at most 32); We1's rows are read through L1 (every lane of a warp reads the
// same rows: broadcasts)
__device__ __forceinline__ void enc_partial32(const __nv_bfloat16 *__restrict__ we1, int m, int64_t col,
                                              const float (&f)[32], int nv, float (&pacc)[32])
{
#pragma unroll
    for (int c = 0; c < 32; ++c) {   // fully unrolled: f is indexed by constants only
        if (c >= nv) break;
        const uint4 *w = reinterpret_cast<const uint4 *>(we1 + (col + c) * m);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            if (8 * q >= m) break;
            const uint4 u = __ldg(w + q);
            const uint32_t ww[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                pacc[8 * q + 2 * e] = fmaf(f[c], __uint_as_float(ww[e] << 16), pacc[8 * q + 2 * e]);
                pacc[8 * q + 2 * e + 1] = fmaf(f[c], __uint_as_float(ww[e] & 0xFFFF0000u), pacc[8 * q + 2 * e + 1]);
            }
        }
    }
}

struct GemmShape {
    int64_t M, N, K;
    int64_t kc;          // K per split, a multiple of 64
    int nm, nn, splits;
    int64_t units;       // nm * nn * splits
};

// BM2: 256-row units, two 128-row A sub-tiles per stage against one B tile, the two halves'
// accumulators side by side in TMEM (one unit at a time: no accumulator double buffering).
// TS: the output tile leaves by TMA stores from shared-memory staging boxes, two per half of the
// epilogue warps (128 rows x 64 columns of bf16, 128-byte swizzle; one fills while the other's
// store reads it), for the products that write T x d bf16 tensors: per-thread 16-byte stores of
// 32 different rows per warp instruction made the epilogue, not the products, set such a
// product's pace.
template <int BN_, bool ALO_ = false, bool BM2_ = false, bool TS_ = false> struct GemmCfg {
    static constexpr int BN = BN_;
    static constexpr uint32_t A_TILE = 128 * 64 * 2;        // 128 rows x 64 K, bf16
    static constexpr uint32_t A_STAGE = A_TILE * (ALO_ ? 2 : 1) * (BM2_ ? 2 : 1);   // hi (+ lo), per half
    static constexpr uint32_t B_STAGE = BN_ * 64 * 2;       // BN rows x 64 K, bf16
    static constexpr uint32_t STAGE = A_STAGE + B_STAGE;
    static constexpr uint32_t STG_HALF = 128 * 64 * 2;      // TS: one staging box
    static constexpr uint32_t STG_BYTES = TS_ ? 4 * STG_HALF : 0;   // two per half
    // 4 stages at BN = 256, 6 at 128 (3, 4 with lo; 3 for BM2); TS: 3 at BN = 256 (2 with lo)
    // beside its four boxes, from a larger share of the 227 KB
    static constexpr int NST = ((TS_ ? 224 : 200) * 1024 - (int)STG_BYTES) / (int)STAGE;
    static constexpr uint32_t OFF_STG = NST * STAGE;        // 1024-aligned (STAGE is)
    static constexpr uint32_t SMEM_BYTES = NST * STAGE + STG_BYTES + 1024;
    static_assert(SMEM_BYTES <= 232448 - 512, "shared memory budget");
    static constexpr uint32_t TMEM_COLS = 2 * BN_;          // two accumulators
    static_assert(TMEM_COLS <= 512, "TMEM budget");
    static constexpr int EPI = 256;                         // epilogue threads (8 warps)
    static constexpr int THREADS = 64 + EPI;
};

__device__ __forceinline__ void gemm_unit(const GemmShape &g, int64_t u, int &mb, int &nb, int &ks)
{
    nb = (int)(u % g.nn);
    const int64_t rest = u / g.nn;
    mb = (int)(rest % g.nm);
    ks = (int)(rest / g.nm);
}

// ---- the epilogue's element-wise steps on 32 consecutive columns of one row ----------------
__device__ __forceinline__ void st_bf16x32(__nv_bfloat16 *dst, const float (&v)[32], int nv)
{
    if (nv == 32) {
        uint4 *o = reinterpret_cast<uint4 *>(dst);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            uint32_t pk[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                __nv_bfloat162 h = __floats2bfloat162_rn(v[8 * q + 2 * e], v[8 * q + 2 * e + 1]);
                pk[e] = *reinterpret_cast<uint32_t *>(&h);
            }
            o[q] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
        }
    } else {   // every index a constant (no dynamic indexing of the register array)
#pragma unroll
        for (int j = 0; j < 32; ++j)
            if (j < nv) dst[j] = __float2bfloat16_rn(v[j]);
    }
}

// hi = v rounded to bf16 at dst, lo = (v - hi) rounded to bf16 at dst_lo (if set)
__device__ __forceinline__ void st_bf16x32_split(__nv_bfloat16 *dst, __nv_bfloat16 *dst_lo, float (&v)[32], int nv)
{
    st_bf16x32(dst, v, nv);
    if (dst_lo) {
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] -= __bfloat162float(__float2bfloat16_rn(v[j]));
        st_bf16x32(dst_lo, v, nv);
    }
}

__device__ __forceinline__ void st_f32x32(float *dst, const float (&v)[32], int nv)
{
    if (nv == 32) {
        float4 *o = reinterpret_cast<float4 *>(dst);
#pragma unroll
        for (int q = 0; q < 8; ++q) o[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
    } else {
#pragma unroll
        for (int j = 0; j < 32; ++j)
            if (j < nv) dst[j] = v[j];
    }
}

__device__ __forceinline__ void ld_bf16x32(const __nv_bfloat16 *src, float (&x)[32], int nv)
{
    if (nv == 32) {
        load_bf16_row<32>(src, x);
    } else {
#pragma unroll
        for (int j = 0; j < 32; ++j) x[j] = j < nv ? __bfloat162float(src[j]) : 0.0f;
    }
}

__device__ __forceinline__ void ld_f32x32(const float *src, float (&x)[32], int nv)
{
    if (nv == 32) {
        const float4 *s = reinterpret_cast<const float4 *>(src);
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const float4 t = s[q];
            x[4 * q] = t.x; x[4 * q + 1] = t.y; x[4 * q + 2] = t.z; x[4 * q + 3] = t.w;
        }
    } else {
#pragma unroll
        for (int j = 0; j < 32; ++j) x[j] = j < nv ? src[j] : 0.0f;
    }
}

// v: the accumulator's columns [col, col + nv) of row `row` (nv <= 32; the vector forms need
// nv == 32 and 16-byte aligned rows, which the host guarantees for nv == 32)
__device__ __forceinline__ void gemm_epilogue(const GemmEp &ep, int64_t row, int64_t col, float (&v)[32], int nv,
                                              int ks)
{
    switch (ep.mode) {
    case GEP_F32:
        st_f32x32(static_cast<float *>(ep.out) + ks * ep.split_stride + row * ep.ldo + col, v, nv);
        break;
    case GEP_BF16:
        st_bf16x32(static_cast<__nv_bfloat16 *>(ep.out) + row * ep.ldo + col, v, nv);
        break;
    case GEP_P_A:
        if (ep.out) st_f32x32(static_cast<float *>(ep.out) + row * ep.ldo + col, v, nv);
        act_fast_row<32>(ep.act, v);
        st_bf16x32_split(static_cast<__nv_bfloat16 *>(ep.out2) + row * ep.ldo2 + col,
                         ep.lo ? ep.lo + row * ep.ldo2 + col : nullptr, v, nv);
        break;
    case GEP_ADD_AUX:
        if (col < ep.aux_cols) {
            const int na = ep.aux_cols - col < nv ? (int)(ep.aux_cols - col) : nv;
            float x[32];
            ld_bf16x32(static_cast<const __nv_bfloat16 *>(ep.aux) + row * ep.lda + col, x, na);
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] = j < na ? v[j] + x[j] : v[j];
        }
        st_bf16x32(static_cast<__nv_bfloat16 *>(ep.out) + row * ep.ldo + col, v, nv);
        break;
    case GEP_ACT:
        if (ep.out2) st_f32x32(static_cast<float *>(ep.out2) + row * ep.ldo2 + col, v, nv);
        act_fast_row<32>(ep.act, v);
        st_bf16x32_split(static_cast<__nv_bfloat16 *>(ep.out) + row * ep.ldo + col,
                         ep.lo ? ep.lo + row * ep.ldo + col : nullptr, v, nv);
        break;
    case GEP_DACT: {
        float x[32], dx[32];
        ld_f32x32(static_cast<const float *>(ep.aux) + row * ep.lda + col, x, nv);
        dact_fast_row<32>(ep.act, x, dx);
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] *= dx[j];
        st_bf16x32_split(static_cast<__nv_bfloat16 *>(ep.out) + row * ep.ldo + col,
                         ep.lo ? ep.lo + row * ep.ldo + col : nullptr, v, nv);
        if (ep.out2) {
            act_fast_row<32>(ep.act, x);
            st_bf16x32(static_cast<__nv_bfloat16 *>(ep.out2) + row * ep.ldo2 + col, x, nv);
        }
        break;
    }
    case GEP_AXPBY: {
        float x[32];
        ld_bf16x32(static_cast<const __nv_bfloat16 *>(ep.aux) + row * ep.lda + col, x, nv);
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] = fmaf(ep.alpha, v[j], ep.beta * x[j]);
        st_bf16x32(static_cast<__nv_bfloat16 *>(ep.out) + row * ep.ldo + col, v, nv);
        break;
    }
    case GEP_DF:
        st_bf16x32(static_cast<__nv_bfloat16 *>(ep.out) + row * ep.ldo + col, v, nv);
        if (ep.rmw && col < ep.aux_cols) {
            const int na = ep.aux_cols - col < nv ? (int)(ep.aux_cols - col) : nv;
            float x[32], y[32];
            __nv_bfloat16 *r = ep.rmw + row * ep.ldr + col;
            ld_bf16x32(r, y, na);
            ld_bf16x32(static_cast<const __nv_bfloat16 *>(ep.aux) + row * ep.lda + col, x, na);
#pragma unroll
            for (int j = 0; j < 32; ++j) y[j] += x[j];
            st_bf16x32(r, y, na);
        }
        break;
    }
}

// TS: the values of an output tile's 32 columns as gemm_epilogue computes them, without its bf16
// store (the caller stages them for a TMA store). Only GEP_BF16, GEP_ADD_AUX and GEP_DF; GEP_DF's
// dX[:, :r] read-modify-write still goes to global memory. in_rows: row < M and col < N.
__device__ __forceinline__ void gemm_epilogue_ts(const GemmEp &ep, int64_t row, int64_t col, float (&v)[32], int nv,
                                                 bool in_rows)
{
    if (!in_rows) return;
    if (ep.mode == GEP_ADD_AUX && col < ep.aux_cols) {
        const int na = ep.aux_cols - col < nv ? (int)(ep.aux_cols - col) : nv;
        float x[32];
        ld_bf16x32(static_cast<const __nv_bfloat16 *>(ep.aux) + row * ep.lda + col, x, na);
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] = j < na ? v[j] + x[j] : v[j];
    } else if (ep.mode == GEP_DF && ep.rmw && col < ep.aux_cols) {
        const int na = ep.aux_cols - col < nv ? (int)(ep.aux_cols - col) : nv;
        float x[32], y[32];
        __nv_bfloat16 *r = ep.rmw + row * ep.ldr + col;
        ld_bf16x32(r, y, na);
        ld_bf16x32(static_cast<const __nv_bfloat16 *>(ep.aux) + row * ep.lda + col, x, na);
#pragma unroll
        for (int j = 0; j < 32; ++j) y[j] += x[j];
        st_bf16x32(r, y, na);
    }
}

// tma_lo: the lo matrix of A (same shape and layout as A; read only with ALO); tmo: the output
// (bf16, N x M, boxes of 64 columns x 128 rows, 128-byte swizzle; read only with TS)
// ENCP: the epilogue of the encoder fused into the FFN down-projection (the GemmEp ENCP fields)
// instead of gemm_epilogue.
// BM2 (GemmCfg): units of 256 rows (two 128-row MMAs per K step sharing the B tile, ~128 flop per
// shared-memory byte against ~85), for long K where a unit's epilogue is short next to its
// products; not with ALO or MC.
// MC: CTA pairs (clusters of 2) take the row blocks 2p and 2p + 1 of the same column block and K
// split; each CTA loads its own A tile and half of the B tile, multicast into both CTAs, so each
// reads 2/3 of a stage's bytes from L2. A stage's `empty` barrier then takes an arrival from both
// CTAs' MMA commits (multicast), so neither refills it before both have read it. (For K-major B
// the tensor map's box is BN / 2 rows.)
template <int BN, bool AMN, bool BMN, bool ALO, bool ENCP = false, bool MC = false, bool BM2 = false,
          bool TS = false>
__global__ void __launch_bounds__(320, 1)
    k_gemm(const __grid_constant__ CUtensorMap tma, const __grid_constant__ CUtensorMap tma_lo,
           const __grid_constant__ CUtensorMap tmb, const __grid_constant__ CUtensorMap tmo, const GemmShape g,
           const GemmEp ep)
{
    using C = GemmCfg<BN, ALO, BM2, TS>;
    static_assert(!(BM2 && (ALO || MC)), "256-row units without hi + lo A or pairs");
    static_assert(!(TS && (ENCP || BM2)), "TMA-store epilogue: plain 128-row units");
    constexpr int MH = BM2 ? 2 : 1;   // 128-row halves per unit (g.nm counts units of 128 * MH rows)
    griddep_wait();               // the previous kernel of the stream has completed
    griddep_launch_dependents();  // the next one may be scheduled on SMs as they free up
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    __shared__ uint64_t full[C::NST], empty[C::NST], acc_full[2], acc_empty[2], done_bar;
    __shared__ uint32_t tmem_base_sh;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    auto k_steps = [&](int ks, int64_t &k0) -> int {
        k0 = (int64_t)ks * g.kc;
        int64_t k1 = k0 + g.kc;
        if (k1 > g.K) k1 = g.K;
        return (int)((k1 - k0 + 63) / 64);
    };
    // this CTA's units: every gridDim.x-th from blockIdx.x, or for a pair every (gridDim.x / 2)-th
    // pair unit from the cluster index, the row block 2 * (pair row block) + rank
    const uint32_t crank = MC ? cluster_rank() : 0u;
    const int64_t u_first = MC ? (int64_t)cluster_index() : (int64_t)blockIdx.x;
    const int64_t u_step = MC ? (int64_t)(gridDim.x / 2) : (int64_t)gridDim.x;
    GemmShape gp = g;
    if (MC) {
        gp.nm = (g.nm + 1) / 2;
        gp.units = (int64_t)gp.nm * gp.nn * gp.splits;
    }
    auto unit_of = [&](int64_t u, int &mb, int &nb, int &ks) {
        gemm_unit(gp, u, mb, nb, ks);
        if (MC) mb = 2 * mb + (int)crank;   // past the last row block: loads read zeros, nothing is stored
    };

    if (threadIdx.x == 0) {
        for (int s = 0; s < C::NST; ++s) {
            mbar_init(smem_u32(&full[s]), 1);
            mbar_init(smem_u32(&empty[s]), MC ? 2 : 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(smem_u32(&acc_full[i]), 1);
            mbar_init(smem_u32(&acc_empty[i]), C::EPI);
        }
        mbar_init(smem_u32(&done_bar), 1);
        fence_mbar_init();
    }
    if (warp == 1) tmem_alloc(smem_u32(&tmem_base_sh), C::TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    if (MC) cluster_sync();   // the peer's barriers exist before anything is multicast to them
    tc_fence_after();
    const uint32_t tmem = tmem_base_sh;

    if (warp == 0) {
        // ---------------- producer ----------------
        if (elect_one()) {
            tma_prefetch_desc(&tma);
            if (ALO) tma_prefetch_desc(&tma_lo);
            tma_prefetch_desc(&tmb);
            uint32_t it = 0;
            bool ok = true;
            for (int64_t u = u_first; u < gp.units && ok; u += u_step) {
                int mb, nb, ks;
                unit_of(u, mb, nb, ks);
                int64_t k0;
                const int nk = k_steps(ks, k0);
                for (int kb = 0; kb < nk; ++kb, ++it) {
                    const uint32_t s = it % C::NST, ph = (it / C::NST) & 1;
                    if (!mbar_wait(smem_u32(&empty[s]), ph ^ 1)) {
                        ok = false;
                        break;
                    }
                    const uint32_t bar = smem_u32(&full[s]);
                    mbar_expect_tx(bar, C::STAGE);
                    const uint32_t adst = smem_u32(smem + s * C::STAGE), bdst = adst + C::A_STAGE;
                    const int32_t kx = (int32_t)(k0 + 64 * kb);
                    if (BM2) {   // the unit's two 128-row A sub-tiles
#pragma unroll
                        for (int h = 0; h < 2; ++h) {
                            const int32_t y = mb * 256 + 128 * h;
                            if (!AMN) {
                                tma_load_2d(adst + h * C::A_TILE, &tma, kx, y, bar);
                            } else {
                                tma_load_2d(adst + h * C::A_TILE, &tma, y, kx, bar);
                                tma_load_2d(adst + h * C::A_TILE + 8192, &tma, y + 64, kx, bar);
                            }
                        }
                    } else if (!AMN) {
                        tma_load_2d(adst, &tma, kx, mb * 128, bar);
                        if (ALO) tma_load_2d(adst + C::A_TILE, &tma_lo, kx, mb * 128, bar);
                    } else {
                        tma_load_2d(adst, &tma, mb * 128, kx, bar);
                        tma_load_2d(adst + 8192, &tma, mb * 128 + 64, kx, bar);
                        if (ALO) {
                            tma_load_2d(adst + C::A_TILE, &tma_lo, mb * 128, kx, bar);
                            tma_load_2d(adst + C::A_TILE + 8192, &tma_lo, mb * 128 + 64, kx, bar);
                        }
                    }
                    if (MC) {   // this CTA's half of B, into both CTAs of the pair
                        if (!BMN) {
                            tma_load_2d_mc(bdst + crank * (BN / 2) * 128, &tmb, kx, nb * BN + (int)crank * (BN / 2), bar, 3);
                        } else {
#pragma unroll
                            for (int j = 0; j < BN / 128; ++j) {
                                const int jj = (int)crank * (BN / 128) + j;
                                tma_load_2d_mc(bdst + jj * 8192, &tmb, nb * BN + 64 * jj, kx, bar, 3);
                            }
                        }
                    } else if (!BMN) {
                        tma_load_2d(bdst, &tmb, kx, nb * BN, bar);
                    } else {
#pragma unroll
                        for (int j = 0; j < BN / 64; ++j) tma_load_2d(bdst + j * 8192, &tmb, nb * BN + 64 * j, kx, bar);
                    }
                }
            }
            // drain the loads still in flight before the CTA may exit (for a pair this includes the
            // peer's multicast halves), and for a pair the last MMA commits of both CTAs on this
            // CTA's stage barriers
            const uint32_t n = it < (uint32_t)C::NST ? it : (uint32_t)C::NST;
            for (uint32_t k = 0; k < n; ++k) {
                const uint32_t j = it - 1 - k;
                mbar_wait(smem_u32(&full[j % C::NST]), (j / C::NST) & 1);
                if (MC && ok) mbar_wait(smem_u32(&empty[j % C::NST]), (j / C::NST) & 1);
            }
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if (elect_one()) {
            constexpr uint32_t idesc = idesc_bf16(128, BN, AMN, BMN);
            // stage-0 descriptors, advanced by (byte offset >> 4) in the start-address field.
            // K-major: rows of 128 bytes (64 K), 8-row groups 1024 bytes apart, a K step of 16 =
            // 32 bytes. MN-major: 64-wide blocks of 64 K rows (8 KB) 8192 bytes apart along M/N,
            // 8-row groups along K 1024 bytes apart, a K step of 16 = 16 rows = 2048 bytes.
            const uint32_t a0 = smem_u32(smem), b0 = a0 + C::A_STAGE;
            const uint64_t ad0 = AMN ? smem_desc(a0, 8192, 1024, kSwz128) : smem_desc(a0, 16, 1024, kSwz128);
            const uint64_t bd0 = BMN ? smem_desc(b0, 8192, 1024, kSwz128) : smem_desc(b0, 16, 1024, kSwz128);
            constexpr uint64_t AK = AMN ? (2048 >> 4) : (32 >> 4);
            constexpr uint64_t BK = BMN ? (2048 >> 4) : (32 >> 4);
            uint32_t it = 0, ti = 0;
            bool ok = true;
            for (int64_t u = u_first; u < gp.units && ok; u += u_step, ++ti) {
                int mb, nb, ks;
                unit_of(u, mb, nb, ks);
                int64_t k0;
                const int nk = k_steps(ks, k0);
                // double-buffered accumulators; BM2: one pair of half accumulators, every unit
                const uint32_t ab = BM2 ? 0u : (ti & 1);
                const uint32_t eph = BM2 ? ((ti & 1) ^ 1) : (((ti >> 1) & 1) ^ 1);
                ok = mbar_wait(smem_u32(&acc_empty[ab]), eph);
                tc_fence_after();
                if (!ok) break;
                const uint32_t d_tmem = tmem + ab * BN;
                for (int kb = 0; kb < nk; ++kb, ++it) {
                    const uint32_t s = it % C::NST, ph = (it / C::NST) & 1;
                    ok = mbar_wait(smem_u32(&full[s]), ph);
                    tc_fence_after();
                    if (!ok) break;
                    const uint64_t so = (uint64_t)((s * C::STAGE) >> 4);
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk) {
                        mma_bf16(d_tmem, ad0 + so + kk * AK, bd0 + so + kk * BK, idesc, kb > 0 || kk > 0);
                        if (ALO) mma_bf16(d_tmem, ad0 + so + (C::A_TILE >> 4) + kk * AK, bd0 + so + kk * BK, idesc, true);
                        if (BM2)   // the second 128-row half into the next BN columns
                            mma_bf16(d_tmem + BN, ad0 + so + (C::A_TILE >> 4) + kk * AK, bd0 + so + kk * BK, idesc,
                                     kb > 0 || kk > 0);
                    }
                    // the stage is free once these MMAs are done (for a pair: once both CTAs' are)
                    if (MC)
                        mma_commit_mc(smem_u32(&empty[s]), 3);
                    else
                        mma_commit(smem_u32(&empty[s]));
                }
                if (!ok) break;
                mma_commit(smem_u32(&acc_full[ab]));
            }
            mma_commit(smem_u32(&done_bar));
            mbar_wait(smem_u32(&done_bar), 0);
        }
    } else {
        // ---------------- epilogue warps ----------------
        const int q = warp & 3;                 // TMEM lane quarter this warp may access
        const int half = (warp - 2) >> 2;       // which half of the BN columns
        const int rin = q * 32 + lane;          // row within the 128-row block
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        uint32_t ti = 0, stg_it = 0;   // units; TS staging boxes filled
        bool ok = true;
        for (int64_t u = u_first; u < gp.units && ok; u += u_step, ++ti) {
            int mb, nb, ks;
            unit_of(u, mb, nb, ks);
            const uint32_t ab = BM2 ? 0u : (ti & 1);
            ok = mbar_wait(smem_u32(&acc_full[ab]), BM2 ? (ti & 1) : ((ti >> 1) & 1));
            tc_fence_after();
            if (!ok) break;
#pragma unroll 1
            for (int h = 0; h < MH; ++h) {   // the unit's 128-row halves (one unless BM2)
                const int64_t row = (int64_t)mb * (128 * MH) + 128 * h + rin;
                const uint32_t acc_col = (ab + (uint32_t)h) * BN;
                float pacc[32];
                if (ENCP) {
#pragma unroll
                    for (int j = 0; j < 32; ++j) pacc[j] = 0.0f;
                }
                if (TS) {
                    // 64 columns at a time through this half's two staging boxes in turn, each
                    // stored by one thread
                    const bool issuer = q == 0 && lane == 0;
#pragma unroll 1
                    for (int c0 = half * (BN / 2); c0 < (half + 1) * (BN / 2); c0 += 64, ++stg_it) {
                        uint8_t *stg = smem + C::OFF_STG + (2 * half + (stg_it & 1)) * C::STG_HALF;
                        if (issuer) bulk_wait_read<1>();   // the box's previous store has read it
                        named_barrier(1 + half, 128);
                        float v2[2][32];
                        tmem_ld32(tmem + lane_base + acc_col + c0, v2[0]);   // warp-collective: every lane
                        tmem_ld32(tmem + lane_base + acc_col + c0 + 32, v2[1]);
                        tmem_ld_wait();
                        tmem_regs_ready(v2[0]);
                        tmem_regs_ready(v2[1]);
#pragma unroll
                        for (int hh = 0; hh < 2; ++hh) {
                            const int64_t col = (int64_t)nb * BN + c0 + 32 * hh;
                            const int nv = g.N - col < 32 ? (int)(g.N - col) : 32;
                            gemm_epilogue_ts(ep, row, col, v2[hh], nv, row < g.M && col < g.N);
                            uint32_t pk[16];
#pragma unroll
                            for (int e = 0; e < 16; ++e) {
                                __nv_bfloat162 b2 = __floats2bfloat162_rn(v2[hh][2 * e], v2[hh][2 * e + 1]);
                                pk[e] = *reinterpret_cast<uint32_t *>(&b2);
                            }
#pragma unroll
                            for (int e = 0; e < 4; ++e)
                                *reinterpret_cast<uint4 *>(stg + swz_offset((uint32_t)rin, 64 * hh + 16 * e, 128)) =
                                    make_uint4(pk[4 * e], pk[4 * e + 1], pk[4 * e + 2], pk[4 * e + 3]);
                        }
                        fence_async_smem();
                        named_barrier(1 + half, 128);
                        const int64_t row0 = (int64_t)mb * (128 * MH) + 128 * h, col0 = (int64_t)nb * BN + c0;
                        if (issuer && row0 < g.M && col0 < g.N) {   // boxes past the tensor: nothing to store
                            tma_store_2d(&tmo, (int32_t)col0, (int32_t)row0, smem_u32(stg));
                            bulk_commit();
                        }
                    }
                }
#pragma unroll 1
                for (int c = half * (BN / 2); c < (TS ? half * (BN / 2) : (half + 1) * (BN / 2)); c += 32) {
                    float v[32];
                    tmem_ld32(tmem + lane_base + acc_col + c, v);   // warp-collective: every lane
                    tmem_ld_wait();
                    tmem_regs_ready<32>(v);
                    const int64_t col = (int64_t)nb * BN + c;
                    if (col < g.N && row < g.M) {
                        const int nv = g.N - col < 32 ? (int)(g.N - col) : 32;
                        if (ENCP) {
                            // F as the FFN's bf16 output, then its share of P = F . We1
#pragma unroll
                            for (int j = 0; j < 32; ++j) v[j] = __bfloat162float(__float2bfloat16_rn(v[j]));
                            if (ep.out) st_bf16x32(static_cast<__nv_bfloat16 *>(ep.out) + row * ep.ldo + col, v, nv);
                            enc_partial32(ep.we1, ep.pm, col, v, nv, pacc);
                        } else {
                            gemm_epilogue(ep, row, col, v, nv, ks);
                        }
                    }
                }
                if (h == MH - 1) {
                    tc_fence_before();
                    mbar_arrive(smem_u32(&acc_empty[ab]));   // this accumulator may be overwritten
                }
                if (ENCP && row < g.M) {
                    float *dst = ep.pslots + (int64_t)(nb * 2 + half) * ep.slot_stride + row * ep.pm;
#pragma unroll
                    for (int q = 0; q < 8; ++q)
                        if (4 * q < ep.pm)
                            reinterpret_cast<float4 *>(dst)[q] =
                                make_float4(pacc[4 * q], pacc[4 * q + 1], pacc[4 * q + 2], pacc[4 * q + 3]);
                }
            }
        }
    }
    if (TS && warp >= 2 && (warp & 3) == 0 && lane == 0) bulk_wait<0>();   // the output tiles' stores are done
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, C::TMEM_COLS);
    }
    if (MC) cluster_sync();   // neither CTA of a pair leaves while the other may still address it
}

// The encoder's end after the fused down-projection, one token row per warp: lane j < m sums
// column j of the row's nslots partial slots in slot order (fp32; the lanes read the slots'
// rows coalesced), saves P if asked, and takes A_j = phi(P_j); lane n < r then forms
// E_n = sum over j of A_j . We2[j][n] (the A_j from lane j by shuffles, j in order) and stores
// B = X[:, :r] + E rounded to bf16. m, r <= 32.
__global__ void __launch_bounds__(256) k_enc_finish(const float *__restrict__ pslots, int nslots, int64_t slot_stride,
                                                    int64_t T, int m, int r, int act, float *__restrict__ P,
                                                    const __nv_bfloat16 *__restrict__ We2,
                                                    const __nv_bfloat16 *__restrict__ X, int64_t ldx,
                                                    __nv_bfloat16 *__restrict__ B)
{
    griddep_wait();
    griddep_launch_dependents();
    const int lane = threadIdx.x & 31;
    const int64_t t = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
    if (t >= T) return;   // whole warps
    float p = 0.0f;
    if (lane < m) {
        const float *src = pslots + t * m + lane;
        for (int s = 0; s < nslots; ++s) p += src[s * slot_stride];
        if (P) P[t * m + lane] = p;
    }
    const float a = lane < m ? act_f(act, p) : 0.0f;
    float e = 0.0f;
    for (int j = 0; j < m; ++j) {
        const float aj = __shfl_sync(0xffffffffu, a, j);
        if (lane < r) e = fmaf(aj, __bfloat162float(We2[j * r + lane]), e);
    }
    if (lane < r) B[t * r + lane] = __float2bfloat16_rn(__bfloat162float(X[t * ldx + lane]) + e);
}

}  // namespace tc
}  // namespace resbm
