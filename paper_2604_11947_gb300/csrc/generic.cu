// generic.cu -- the portable CUDA-core path of the ResBM boundary bottleneck.
//
// Every product of Sec. 3.2 (and of its chain-rule backward) runs through one tiled FFMA
// kernel whose operand loaders and epilogue are small functors: the nonlinearity, its
// derivative, the identity-path add of Eq. generalized_transformer_equation and the rounding
// to the I/O dtype are folded into loads and stores. It handles every shape and both dtypes
// and is the fp32 path (fp32 products at full fp32 precision). Weight gradients are split
// over tokens into fp32 partials that a second kernel sums in a fixed order (deterministic).
#include <type_traits>

#include "common.cuh"
#include "internal.h"

namespace resbm {
namespace {

constexpr int BM = 64, BN = 64, BK = 16, NT = 256;

// ---- operand loaders: element (row, col) of a logical matrix as fp32 -----------------------
template <typename T> struct LdRM {  // M[row][col] = p[row * ld + col]
    const T *p; int64_t ld;
    __device__ float operator()(int64_t i, int64_t k) const { return to_f32(p[i * ld + k]); }
};
template <typename T> struct LdT {   // M[row][col] = p[col * ld + row] (transposed view)
    const T *p; int64_t ld;
    __device__ float operator()(int64_t i, int64_t k) const { return to_f32(p[k * ld + i]); }
};
struct LdAct {                       // phi(p[row][col])
    const float *p; int64_t ld; int act;
    __device__ float operator()(int64_t i, int64_t k) const { return act_f(act, p[i * ld + k]); }
};
struct LdActT {                      // phi(p[col][row])
    const float *p; int64_t ld; int act;
    __device__ float operator()(int64_t i, int64_t k) const { return act_f(act, p[k * ld + i]); }
};
struct LdDact {                      // g[row][col] * phi'(x[row][col])
    const float *g; const float *x; int64_t ld; int act;
    __device__ float operator()(int64_t i, int64_t k) const
    {
        return g[i * ld + k] * dact_f(act, x[i * ld + k]);
    }
};

// ---- epilogues: ep(row, col, split, acc) ----------------------------------------------------
struct EpF32 {
    float *out; int64_t ld; int64_t zstride;
    __device__ void operator()(int64_t i, int64_t n, int z, float acc) const
    {
        out[z * zstride + i * ld + n] = acc;
    }
};
template <typename T> struct EpStore {
    T *out; int64_t ld;
    __device__ void operator()(int64_t i, int64_t n, int, float acc) const
    {
        out[i * ld + n] = from_f32<T>(acc);
    }
};
template <typename T> struct EpEncB {   // B = X . I_{d x r} + E
    T *B; const T *X; int64_t r, d;
    __device__ void operator()(int64_t i, int64_t n, int, float acc) const
    {
        B[i * r + n] = from_f32<T>(to_f32(X[i * d + n]) + acc);
    }
};
template <typename T> struct EpDecY {   // Y = [merge] B . I_{r x d} + D
    T *Y; const T *B; int64_t d, r; int merge;
    __device__ void operator()(int64_t i, int64_t n, int, float acc) const
    {
        const float skip = (merge && n < r) ? to_f32(B[i * r + n]) : 0.0f;
        Y[i * d + n] = from_f32<T>(skip + acc);
    }
};
template <typename T> struct EpDecDB {  // dB = [merge] dY . I_{r x d}^T + dQ . Wd1^T
    T *dB; const T *dY; int64_t r, d; int merge;
    __device__ void operator()(int64_t i, int64_t n, int, float acc) const
    {
        const float skip = merge ? to_f32(dY[i * d + n]) : 0.0f;
        dB[i * r + n] = from_f32<T>(skip + acc);
    }
};

// C[M x N] = A[M x K] . B[K x N]; blockIdx.z selects a K range of length kchunk.
template <class LA, class LB, class EP>
__global__ void __launch_bounds__(NT) k_gemm(int64_t M, int64_t N, int64_t K, int64_t kchunk,
                                             LA la, LB lb, EP ep)
{
    __shared__ float As[BK][BM + 1];
    __shared__ float Bs[BK][BN + 1];
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int64_t m0 = (int64_t)blockIdx.x * BM, n0 = (int64_t)blockIdx.y * BN;
    const int64_t kb0 = (int64_t)blockIdx.z * kchunk;
    const int64_t kb1 = min(K, kb0 + kchunk);
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = 0.0f;

    for (int64_t k0 = kb0; k0 < kb1; k0 += BK) {
        for (int e = tid; e < BM * BK; e += NT) {
            const int kk = e % BK, mm = e / BK;
            const int64_t gm = m0 + mm, gk = k0 + kk;
            As[kk][mm] = (gm < M && gk < kb1) ? la(gm, gk) : 0.0f;
        }
        for (int e = tid; e < BN * BK; e += NT) {
            const int nn = e % BN, kk = e / BN;
            const int64_t gn = n0 + nn, gk = k0 + kk;
            Bs[kk][nn] = (gn < N && gk < kb1) ? lb(gk, gn) : 0.0f;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < BK; ++kk) {
            float a[4], b[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) a[i] = As[kk][ty + 16 * i];
#pragma unroll
            for (int j = 0; j < 4; ++j) b[j] = Bs[kk][tx + 16 * j];
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int64_t gm = m0 + ty + 16 * i, gn = n0 + tx + 16 * j;
            if (gm < M && gn < N) ep(gm, gn, (int)blockIdx.z, acc[i][j]);
        }
}

template <class LA, class LB, class EP>
cudaError_t gemm(int64_t M, int64_t N, int64_t K, int splits, LA la, LB lb, EP ep,
                 cudaStream_t s)
{
    if (M <= 0 || N <= 0) return cudaSuccess;
    int64_t kchunk = K;
    if (splits > 1) kchunk = ((K + splits - 1) / splits + BK - 1) / BK * BK;
    if (kchunk <= 0) kchunk = BK;
    const int64_t nz = (K + kchunk - 1) / kchunk;
    dim3 grid((unsigned)((M + BM - 1) / BM), (unsigned)((N + BN - 1) / BN),
              (unsigned)(nz > 0 ? nz : 1));
    k_gemm<<<grid, NT, 0, s>>>(M, N, K, kchunk, la, lb, ep);
    count_launches(1);
    return cudaGetLastError();
}

// out[e] = sum over s = 0, 1, ..., S-1 of part[s * n + e]   (fixed order)
__global__ void k_reduce_splits(const float *__restrict__ part, int64_t n, int S,
                                float *__restrict__ out)
{
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < n;
         e += (int64_t)gridDim.x * blockDim.x) {
        float acc = 0.0f;
        for (int s = 0; s < S; ++s) acc += part[s * n + e];
        out[e] = acc;
    }
}

// dX[:, :r] += dB  (the gradient of the truncating identity projection)
template <typename T>
__global__ void k_dx_accumulate(T *dX, const T *__restrict__ dB, int64_t Tn, int64_t d, int64_t r)
{
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < Tn * r;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int64_t t = e / r, j = e - t * r;
        dX[t * d + j] = from_f32<T>(to_f32(dX[t * d + j]) + to_f32(dB[e]));
    }
}

// out = the n x n identity matrix
template <typename T> __global__ void k_identity(T *out, int64_t n)
{
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < n * n; e += (int64_t)gridDim.x * blockDim.x)
        out[e] = from_f32<T>(e / n == e % n ? 1.0f : 0.0f);
}

int grid_for(int64_t n, const Ctx &c)
{
    int64_t g = (n + 255) / 256;
    const int64_t cap = (int64_t)c.sm_count * 8;
    if (g > cap) g = cap;
    return (int)(g < 1 ? 1 : g);
}

// Token splits of the weight-gradient reductions.
int token_splits(int64_t T)
{
    int64_t s = (T + 1023) / 1024;
    if (s < 1) s = 1;
    if (s > 32) s = 32;
    return (int)s;
}

// A weight gradient over tokens: partials (if split) then a fixed-order sum.
template <class LA, class LB>
cudaError_t weight_grad(int64_t M, int64_t N, int64_t T, LA la, LB lb, float *out, float *part,
                        const Ctx &c)
{
    const int S = token_splits(T);
    if (S == 1) return gemm(M, N, T, 1, la, lb, EpF32{out, N, 0}, c.stream);
    cudaError_t e = gemm(M, N, T, S, la, lb, EpF32{part, N, M * N}, c.stream);
    if (e != cudaSuccess) return e;
    // the number of splits actually launched (the last ones may be empty)
    int64_t kchunk = ((T + S - 1) / S + BK - 1) / BK * BK;
    const int nz = (int)((T + kchunk - 1) / kchunk);
    k_reduce_splits<<<grid_for(M * N, c), 256, 0, c.stream>>>(part, M * N, nz, out);
    count_launches(1);
    return cudaGetLastError();
}

struct GenericWs {
    float *P, *Q, *dG, *dA, *part1, *part2;
};

GenericWs carve(const resbm_desc &d, int op, void *base, size_t *bytes)
{
    WsCarver w(base);
    GenericWs g{};
    const int64_t T = d.T, S = token_splits(d.T);
    switch (op) {
    case RESBM_OP_ENCODE_FWD:
        g.P = w.take<float>(T * d.m);
        break;
    case RESBM_OP_DECODE_FWD:
        g.Q = w.take<float>(T * d.m);
        break;
    case RESBM_OP_DECODE_BWD:
        g.Q = w.take<float>(T * d.m);
        g.dG = w.take<float>(T * d.m);
        g.part1 = w.take<float>(S * d.m * d.d);
        g.part2 = w.take<float>(S * d.r * d.m);
        break;
    case RESBM_OP_ENCODE_BWD:
        g.P = w.take<float>(T * d.m);
        g.dA = w.take<float>(T * d.m);
        g.part1 = w.take<float>(S * d.d * d.m);
        g.part2 = w.take<float>(S * d.m * d.r);
        break;
    default:
        break;
    }
    if (bytes) *bytes = w.used;
    return g;
}

template <typename T>
cudaError_t enc_fwd_t(const resbm_desc &d, const T *X, const T *F, const T *We1, const T *We2,
                      T *B, float *P_save, void *ws, const Ctx &c)
{
    GenericWs g = carve(d, RESBM_OP_ENCODE_FWD, ws, nullptr);
    float *P = P_save ? P_save : g.P;
    cudaError_t e = gemm(d.T, d.m, d.d, 1, LdRM<T>{F, d.d}, LdRM<T>{We1, d.m},
                         EpF32{P, d.m, 0}, c.stream);                       // P = F . We1
    if (e != cudaSuccess) return e;
    return gemm(d.T, d.r, d.m, 1, LdAct{P, d.m, d.act}, LdRM<T>{We2, d.r},
                EpEncB<T>{B, X, d.r, d.d}, c.stream);                       // B = X I + phi(P) We2
}

template <typename T>
cudaError_t dec_fwd_t(const resbm_desc &d, const T *B, const T *Wd1, const T *Wd2, T *Y,
                      void *ws, const Ctx &c)
{
    GenericWs g = carve(d, RESBM_OP_DECODE_FWD, ws, nullptr);
    cudaError_t e = gemm(d.T, d.m, d.r, 1, LdRM<T>{B, d.r}, LdRM<T>{Wd1, d.m},
                         EpF32{g.Q, d.m, 0}, c.stream);                     // Q = B . Wd1
    if (e != cudaSuccess) return e;
    return gemm(d.T, d.d, d.m, 1, LdAct{g.Q, d.m, d.act}, LdRM<T>{Wd2, d.d},
                EpDecY<T>{Y, B, d.d, d.r, d.merge_identity}, c.stream);     // Y = [B I] + phi(Q) Wd2
}

template <typename T>
cudaError_t dec_bwd_t(const resbm_desc &d, const T *dY, const T *B, const T *Wd1, const T *Wd2,
                      T *dB, float *dWd1, float *dWd2, void *ws, const Ctx &c)
{
    GenericWs g = carve(d, RESBM_OP_DECODE_BWD, ws, nullptr);
    cudaError_t e = gemm(d.T, d.m, d.r, 1, LdRM<T>{B, d.r}, LdRM<T>{Wd1, d.m},
                         EpF32{g.Q, d.m, 0}, c.stream);                     // Q = B . Wd1
    if (e != cudaSuccess) return e;
    e = gemm(d.T, d.m, d.d, 1, LdRM<T>{dY, d.d}, LdT<T>{Wd2, d.d}, EpF32{g.dG, d.m, 0},
             c.stream);                                                     // dG = dY . Wd2^T
    if (e != cudaSuccess) return e;
    const LdDact dQ{g.dG, g.Q, d.m, d.act};                                 // dQ = dG * phi'(Q)
    e = gemm(d.T, d.r, d.m, 1, dQ, LdT<T>{Wd1, d.m},
             EpDecDB<T>{dB, dY, d.r, d.d, d.merge_identity}, c.stream);     // dB
    if (e != cudaSuccess) return e;
    e = weight_grad(d.m, d.d, d.T, LdActT{g.Q, d.m, d.act}, LdRM<T>{dY, d.d}, dWd2, g.part1,
                    c);                                                     // dWd2 = phi(Q)^T dY
    if (e != cudaSuccess) return e;
    return weight_grad(d.r, d.m, d.T, LdT<T>{B, d.r}, dQ, dWd1, g.part2, c); // dWd1 = B^T dQ
}

template <typename T>
cudaError_t enc_bwd_t(const resbm_desc &d, const T *dB, const T *F, const float *P_save,
                      const T *We1, const T *We2, T *dF, T *dX, float *dWe1, float *dWe2,
                      void *ws, const Ctx &c)
{
    GenericWs g = carve(d, RESBM_OP_ENCODE_BWD, ws, nullptr);
    cudaError_t e = cudaSuccess;
    const float *P = P_save;
    if (!P) {
        e = gemm(d.T, d.m, d.d, 1, LdRM<T>{F, d.d}, LdRM<T>{We1, d.m}, EpF32{g.P, d.m, 0},
                 c.stream);                                                 // P = F . We1
        if (e != cudaSuccess) return e;
        P = g.P;
    }
    e = gemm(d.T, d.m, d.r, 1, LdRM<T>{dB, d.r}, LdT<T>{We2, d.r}, EpF32{g.dA, d.m, 0},
             c.stream);                                                     // dA = dB . We2^T
    if (e != cudaSuccess) return e;
    const LdDact dP{g.dA, P, d.m, d.act};                                   // dP = dA * phi'(P)
    e = gemm(d.T, d.d, d.m, 1, dP, LdT<T>{We1, d.m}, EpStore<T>{dF, d.d}, c.stream); // dF
    if (e != cudaSuccess) return e;
    e = weight_grad(d.d, d.m, d.T, LdT<T>{F, d.d}, dP, dWe1, g.part1, c);   // dWe1 = F^T dP
    if (e != cudaSuccess) return e;
    e = weight_grad(d.m, d.r, d.T, LdActT{P, d.m, d.act}, LdRM<T>{dB, d.r}, dWe2, g.part2,
                    c);                                                     // dWe2 = phi(P)^T dB
    if (e != cudaSuccess) return e;
    if (dX) {
        k_dx_accumulate<T><<<grid_for(d.T * d.r, c), 256, 0, c.stream>>>(dX, dB, d.T, d.d, d.r);
        count_launches(1);
        e = cudaGetLastError();
    }
    return e;
}

// RMSNorm of every row of Y (the next block's pre-attention norm, after the decoder on the paths
// without the fused form): N = Y / sqrt(mean_j Y_j^2 + eps) * gamma. One warp per row; the squares
// of the stored values summed per lane over a fixed column stride, then by a fixed shuffle tree
// (deterministic). fp32 rows sum in double (their tolerance is fp32's), bf16 rows in float.
template <typename E>
__global__ void __launch_bounds__(256) k_rmsnorm(const E *__restrict__ Y, const E *__restrict__ gamma, float eps,
                                                 int64_t rows, int64_t d, E *__restrict__ N)
{
    using Acc = typename std::conditional<std::is_same<E, float>::value, double, float>::type;
    const int lane = threadIdx.x & 31;
    for (int64_t t = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5); t < rows; t += (int64_t)gridDim.x * 8) {
        const E *y = Y + t * d;
        Acc s = 0;
        for (int64_t j = lane; j < d; j += 32) {
            const Acc v = (Acc)to_f32(y[j]);
            s += v * v;
        }
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        const Acc rstd = (Acc)1 / sqrt(s / (Acc)d + (Acc)eps);
        for (int64_t j = lane; j < d; j += 32)
            N[t * d + j] = from_f32<E>((float)((Acc)to_f32(y[j]) * rstd * (Acc)to_f32(gamma[j])));
    }
}

// Backward of N = RMSNorm(Y) * gamma with the residual stream's own gradient added:
//   dY_out = dY + s g - Y (s^3 / d) sum_j g_j Y_j,  g = dN * gamma,  s = 1 / sqrt(mean_j Y_j^2 + eps)
//   dgamma partial of this block = sum over its rows of dN * Y * s
// A block takes a fixed contiguous range of rows, one row at a time: its threads cover the row's
// columns (vectors of V elements, thread q owning vectors q, q + 256, ...), the two row sums go
// through a fixed shuffle tree and the eight warps' partials in warp order, and each thread keeps
// the dgamma sums of the columns it owns in shared memory (no two threads touch a column), so the
// result does not depend on timing or on the device. The second pass over the row re-reads it
// (from L1 / L2). dY may equal dY_out (read before written by the same thread) or be null.
constexpr int kNormBwdBlocks = 1024;   // ~7 resident per SM on 152 SMs: rows in flight hide the load latency
constexpr int kNormBwdMaxD = 16384;

template <typename E, int V> struct VecOf;
template <> struct VecOf<__nv_bfloat16, 8> {
    static __device__ void unpack(const uint4 u, float *f)
    {
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            f[2 * i] = __uint_as_float(w[i] << 16);
            f[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
        }
    }
    static __device__ void load(const __nv_bfloat16 *p, float *f)
    {
        const uint4 u = *reinterpret_cast<const uint4 *>(p);
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            f[2 * i] = __uint_as_float(w[i] << 16);
            f[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
        }
    }
    static __device__ void store(__nv_bfloat16 *p, const float *f)
    {
        uint32_t w[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            __nv_bfloat162 h = __floats2bfloat162_rn(f[2 * i], f[2 * i + 1]);
            w[i] = *reinterpret_cast<uint32_t *>(&h);
        }
        *reinterpret_cast<uint4 *>(p) = make_uint4(w[0], w[1], w[2], w[3]);
    }
};
template <> struct VecOf<float, 4> {
    static __device__ void unpack(const uint4 u, float *f)
    {
        f[0] = __uint_as_float(u.x); f[1] = __uint_as_float(u.y); f[2] = __uint_as_float(u.z); f[3] = __uint_as_float(u.w);
    }
    static __device__ void load(const float *p, float *f)
    {
        const float4 u = *reinterpret_cast<const float4 *>(p);
        f[0] = u.x; f[1] = u.y; f[2] = u.z; f[3] = u.w;
    }
    static __device__ void store(float *p, const float *f) { *reinterpret_cast<float4 *>(p) = make_float4(f[0], f[1], f[2], f[3]); }
};
template <typename E> struct VecOf<E, 1> {
    static __device__ void load(const E *p, float *f) { f[0] = to_f32(*p); }
    static __device__ void store(E *p, const float *f) { *p = from_f32<E>(f[0]); }
};

template <typename E, int V>
__global__ void __launch_bounds__(256) k_rmsnorm_bwd(const E *__restrict__ Y, const E *__restrict__ gamma, float eps,
                                                     const E *__restrict__ dN, const E *dY, E *dYo,
                                                     float *__restrict__ dg_part, int64_t rows, int64_t d)
{
    extern __shared__ float dgs[];   // d: this block's dgamma sums, column j owned by thread (j / V) % 256
    __shared__ float2 part[2][8];
    using L = VecOf<E, V>;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int64_t nv = d / V;
    for (int64_t q = tid; q < nv; q += 256)
#pragma unroll
        for (int i = 0; i < V; ++i) dgs[q * V + i] = 0.0f;
    const int64_t r0 = rows * blockIdx.x / gridDim.x, r1 = rows * (blockIdx.x + 1) / gridDim.x;
    for (int64_t t = r0; t < r1; ++t) {
        const E *y = Y + t * d, *dn = dN + t * d;
        float sy = 0.0f, sg = 0.0f;   // sum Y^2, sum g Y over this thread's columns
        for (int64_t q = tid; q < nv; q += 256) {
            float a[V], b[V], gm[V];
            L::load(y + q * V, a);
            L::load(dn + q * V, b);
            L::load(gamma + q * V, gm);
#pragma unroll
            for (int i = 0; i < V; ++i) {
                sy = fmaf(a[i], a[i], sy);
                sg = fmaf(b[i] * gm[i], a[i], sg);
            }
        }
        for (int o = 16; o > 0; o >>= 1) {
            sy += __shfl_xor_sync(0xffffffffu, sy, o);
            sg += __shfl_xor_sync(0xffffffffu, sg, o);
        }
        const int pb = (int)((t - r0) & 1);
        if (lane == 0) part[pb][warp] = make_float2(sy, sg);
        __syncthreads();
        float Sy = 0.0f, Sg = 0.0f;
#pragma unroll
        for (int w = 0; w < 8; ++w) {
            Sy += part[pb][w].x;
            Sg += part[pb][w].y;
        }
        const float s = 1.0f / sqrtf(Sy / (float)d + eps);
        const float k = s * s * s * Sg / (float)d;
        for (int64_t q = tid; q < nv; q += 256) {
            float a[V], b[V], gm[V], o[V];
            L::load(y + q * V, a);
            L::load(dn + q * V, b);
            L::load(gamma + q * V, gm);
            if (dY) L::load(dY + t * d + q * V, o);
            else
#pragma unroll
                for (int i = 0; i < V; ++i) o[i] = 0.0f;
            float acc[V];
            if (V % 4 == 0) {   // 16-byte shared accesses: consecutive threads, consecutive chunks
#pragma unroll
                for (int i = 0; i < V; i += 4) {
                    const float4 u = *reinterpret_cast<const float4 *>(dgs + q * V + i);
                    acc[i] = u.x; acc[i + 1] = u.y; acc[i + 2] = u.z; acc[i + 3] = u.w;
                }
            } else {
#pragma unroll
                for (int i = 0; i < V; ++i) acc[i] = dgs[q * V + i];
            }
#pragma unroll
            for (int i = 0; i < V; ++i) {
                o[i] += s * (b[i] * gm[i]) - a[i] * k;
                acc[i] = fmaf(b[i], a[i] * s, acc[i]);
            }
            if (V % 4 == 0) {
#pragma unroll
                for (int i = 0; i < V; i += 4)
                    *reinterpret_cast<float4 *>(dgs + q * V + i) = make_float4(acc[i], acc[i + 1], acc[i + 2], acc[i + 3]);
            } else {
#pragma unroll
                for (int i = 0; i < V; ++i) dgs[q * V + i] = acc[i];
            }
            L::store(dYo + t * d + q * V, o);
        }
    }
    __syncthreads();
    for (int64_t j = tid; j < d; j += 256) dg_part[(int64_t)blockIdx.x * d + j] = dgs[j];
}

// The vector path for rows of at most 256 * KV vectors: each thread keeps its vectors of Y, dN and
// dY (as loaded, 16 bytes each) in registers from the first pass to the second, so a row costs one
// trip to memory, and loads dY with Y and dN. The same sums in the same order as k_rmsnorm_bwd, so
// the same bits.
template <typename E, int V, int KV>
__global__ void __launch_bounds__(256) k_rmsnorm_bwd_reg(const E *__restrict__ Y, const E *__restrict__ gamma, float eps,
                                                         const E *__restrict__ dN, const E *dY, E *dYo,
                                                         float *__restrict__ dg_part, int64_t rows, int64_t d)
{
    extern __shared__ float dgs[];
    __shared__ float2 part[2][8];
    using L = VecOf<E, V>;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int64_t nv = d / V;
#pragma unroll
    for (int k = 0; k < KV; ++k) {
        const int64_t q = tid + 256 * k;
        if (q < nv)
#pragma unroll
            for (int i = 0; i < V; ++i) dgs[q * V + i] = 0.0f;
    }
    const int64_t r0 = rows * blockIdx.x / gridDim.x, r1 = rows * (blockIdx.x + 1) / gridDim.x;
    for (int64_t t = r0; t < r1; ++t) {
        uint4 ry[KV], rn[KV], ro[KV];
#pragma unroll
        for (int k = 0; k < KV; ++k) {   // every load of the row in flight before the first use
            const int64_t q = tid + 256 * k;
            if (q < nv) {
                ry[k] = *reinterpret_cast<const uint4 *>(Y + t * d + q * V);
                rn[k] = *reinterpret_cast<const uint4 *>(dN + t * d + q * V);
                ro[k] = dY ? *reinterpret_cast<const uint4 *>(dY + t * d + q * V) : make_uint4(0u, 0u, 0u, 0u);
            }
        }
        float sy = 0.0f, sg = 0.0f;
#pragma unroll
        for (int k = 0; k < KV; ++k) {
            const int64_t q = tid + 256 * k;
            if (q < nv) {
                float a[V], b[V], gm[V];
                L::unpack(ry[k], a);
                L::unpack(rn[k], b);
                L::load(gamma + q * V, gm);
#pragma unroll
                for (int i = 0; i < V; ++i) {
                    sy = fmaf(a[i], a[i], sy);
                    sg = fmaf(b[i] * gm[i], a[i], sg);
                }
            }
        }
        for (int o = 16; o > 0; o >>= 1) {
            sy += __shfl_xor_sync(0xffffffffu, sy, o);
            sg += __shfl_xor_sync(0xffffffffu, sg, o);
        }
        const int pb = (int)((t - r0) & 1);
        if (lane == 0) part[pb][warp] = make_float2(sy, sg);
        __syncthreads();
        float Sy = 0.0f, Sg = 0.0f;
#pragma unroll
        for (int w = 0; w < 8; ++w) {
            Sy += part[pb][w].x;
            Sg += part[pb][w].y;
        }
        const float s = 1.0f / sqrtf(Sy / (float)d + eps);
        const float kk = s * s * s * Sg / (float)d;
#pragma unroll
        for (int k = 0; k < KV; ++k) {
            const int64_t q = tid + 256 * k;
            if (q < nv) {
                float a[V], b[V], gm[V], o[V], acc[V];
                L::unpack(ry[k], a);
                L::unpack(rn[k], b);
                L::unpack(ro[k], o);
                L::load(gamma + q * V, gm);
#pragma unroll
                for (int i = 0; i < V; i += 4) {
                    const float4 u = *reinterpret_cast<const float4 *>(dgs + q * V + i);
                    acc[i] = u.x; acc[i + 1] = u.y; acc[i + 2] = u.z; acc[i + 3] = u.w;
                }
#pragma unroll
                for (int i = 0; i < V; ++i) {
                    o[i] += s * (b[i] * gm[i]) - a[i] * kk;
                    acc[i] = fmaf(b[i], a[i] * s, acc[i]);
                }
#pragma unroll
                for (int i = 0; i < V; i += 4)
                    *reinterpret_cast<float4 *>(dgs + q * V + i) = make_float4(acc[i], acc[i + 1], acc[i + 2], acc[i + 3]);
                L::store(dYo + t * d + q * V, o);
            }
        }
    }
    __syncthreads();
    for (int64_t j = tid; j < d; j += 256) dg_part[(int64_t)blockIdx.x * d + j] = dgs[j];
}

// dgamma[j] = the blocks' partials summed by a fixed two-level tree: warp w of a CTA sums the
// partials of blocks [w G, (w + 1) G) in block order (eight loads in flight) for the CTA's 32
// columns, then the eight group sums are added in group order. CTA x covers columns 32 x .. + 31.
__global__ void __launch_bounds__(256) k_rmsnorm_dgamma(const float *__restrict__ dg_part, int nblocks, int64_t d,
                                                        float *__restrict__ dgamma)
{
    __shared__ float gs[8][32];
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const int64_t j = (int64_t)blockIdx.x * 32 + lane;
    const int G = (nblocks + 7) / 8;
    const int b0 = w * G, b1 = b0 + G < nblocks ? b0 + G : nblocks;
    float a = 0.0f;
    if (j < d) {
        int b = b0;
        for (; b + 8 <= b1; b += 8) {
            float x[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) x[u] = dg_part[(int64_t)(b + u) * d + j];
#pragma unroll
            for (int u = 0; u < 8; ++u) a += x[u];
        }
        for (; b < b1; ++b) a += dg_part[(int64_t)b * d + j];
    }
    gs[w][lane] = a;
    __syncthreads();
    if (w == 0 && j < d) {
        float t = 0.0f;
#pragma unroll
        for (int g = 0; g < 8; ++g) t += gs[g][lane];
        dgamma[j] = t;
    }
}

}  // namespace

int rmsnorm_bwd_blocks(int64_t rows) { return (int)(rows < kNormBwdBlocks ? (rows < 1 ? 1 : rows) : kNormBwdBlocks); }
bool rmsnorm_bwd_supported(const resbm_desc &d) { return d.d >= 1 && d.d <= kNormBwdMaxD; }
size_t rmsnorm_bwd_ws_bytes(const resbm_desc &d) { return (size_t)rmsnorm_bwd_blocks(d.T) * (size_t)d.d * sizeof(float); }

cudaError_t generic_rmsnorm_bwd(const resbm_desc &d, const void *Y, const void *gamma, float eps, const void *dN,
                                const void *dY, void *dY_out, float *dgamma, void *ws, const Ctx &c)
{
    const int nb = rmsnorm_bwd_blocks(d.T);
    float *part = static_cast<float *>(ws);
    const size_t smem = (size_t)d.d * sizeof(float);
    auto al = [](const void *p) { return p == nullptr || (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
    const bool vec = al(Y) && al(gamma) && al(dN) && al(dY) && al(dY_out) &&
                     d.d % (d.dtype == RESBM_F32 ? 4 : 8) == 0;
    cudaError_t e = cudaSuccess;
    if (d.T > 0) {
        // the register-cached vector path up to 4 vectors a thread (bf16 d <= 8192, fp32 d <= 4096)
        const int64_t nv = d.d / (d.dtype == RESBM_F32 ? 4 : 8);
        const int kv = !vec ? 0 : nv <= 256 ? 1 : nv <= 512 ? 2 : nv <= 1024 ? 4 : 0;
        if (d.dtype == RESBM_F32) {
            auto k = kv == 1 ? k_rmsnorm_bwd_reg<float, 4, 1> : kv == 2 ? k_rmsnorm_bwd_reg<float, 4, 2>
                   : kv == 4 ? k_rmsnorm_bwd_reg<float, 4, 4> : vec ? k_rmsnorm_bwd<float, 4> : k_rmsnorm_bwd<float, 1>;
            e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (e == cudaSuccess)
                k<<<nb, 256, smem, c.stream>>>((const float *)Y, (const float *)gamma, eps, (const float *)dN,
                                              (const float *)dY, (float *)dY_out, part, d.T, d.d);
        } else {
            using bf = __nv_bfloat16;
            auto k = kv == 1 ? k_rmsnorm_bwd_reg<bf, 8, 1> : kv == 2 ? k_rmsnorm_bwd_reg<bf, 8, 2>
                   : kv == 4 ? k_rmsnorm_bwd_reg<bf, 8, 4> : vec ? k_rmsnorm_bwd<bf, 8> : k_rmsnorm_bwd<bf, 1>;
            e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (e == cudaSuccess)
                k<<<nb, 256, smem, c.stream>>>((const bf *)Y, (const bf *)gamma, eps, (const bf *)dN, (const bf *)dY,
                                              (bf *)dY_out, part, d.T, d.d);
        }
        count_launches(1);
        if (e == cudaSuccess) e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    const int64_t gb = (d.d + 31) / 32;
    if (d.T > 0) {
        k_rmsnorm_dgamma<<<(unsigned)gb, 256, 0, c.stream>>>(part, nb, d.d, dgamma);
    } else {
        e = cudaMemsetAsync(dgamma, 0, (size_t)d.d * sizeof(float), c.stream);
        if (e != cudaSuccess) return e;
    }
    count_launches(d.T > 0 ? 1 : 0);
    return cudaGetLastError();
}

cudaError_t generic_rmsnorm(const resbm_desc &d, const void *Y, const void *gamma, float eps, void *N,
                            const Ctx &c)
{
    if (d.T == 0) return cudaSuccess;
    int64_t blocks = (d.T + 7) / 8;
    const int64_t cap = (int64_t)c.sm_count * 16;
    if (blocks > cap) blocks = cap;
    if (d.dtype == RESBM_F32)
        k_rmsnorm<float><<<(unsigned)blocks, 256, 0, c.stream>>>((const float *)Y, (const float *)gamma, eps, d.T, d.d,
                                                                 (float *)N);
    else
        k_rmsnorm<__nv_bfloat16><<<(unsigned)blocks, 256, 0, c.stream>>>(
            (const __nv_bfloat16 *)Y, (const __nv_bfloat16 *)gamma, eps, d.T, d.d, (__nv_bfloat16 *)N);
    count_launches(1);
    return cudaGetLastError();
}

size_t generic_ws_bytes(const resbm_desc &d, int op)
{
    size_t b = 0;
    carve(d, op, nullptr, &b);
    return b;
}

#define RESBM_DISPATCH(dt, F32CALL, BF16CALL) \
    ((dt) == RESBM_F32 ? (F32CALL) : (BF16CALL))

cudaError_t generic_encode_fwd(const resbm_desc &d, const void *X, const void *F, const void *We1,
                               const void *We2, void *B, float *P_save, void *ws, const Ctx &c)
{
    using bf = __nv_bfloat16;
    return RESBM_DISPATCH(d.dtype,
        enc_fwd_t<float>(d, (const float *)X, (const float *)F, (const float *)We1,
                         (const float *)We2, (float *)B, P_save, ws, c),
        enc_fwd_t<bf>(d, (const bf *)X, (const bf *)F, (const bf *)We1, (const bf *)We2,
                      (bf *)B, P_save, ws, c));
}

cudaError_t generic_decode_fwd(const resbm_desc &d, const void *B, const void *Wd1,
                               const void *Wd2, void *Y, void *ws, const Ctx &c)
{
    using bf = __nv_bfloat16;
    return RESBM_DISPATCH(d.dtype,
        dec_fwd_t<float>(d, (const float *)B, (const float *)Wd1, (const float *)Wd2,
                         (float *)Y, ws, c),
        dec_fwd_t<bf>(d, (const bf *)B, (const bf *)Wd1, (const bf *)Wd2, (bf *)Y, ws, c));
}

cudaError_t generic_decode_bwd(const resbm_desc &d, const void *dY, const void *B,
                               const void *Wd1, const void *Wd2, void *dB, float *dWd1,
                               float *dWd2, void *ws, const Ctx &c)
{
    using bf = __nv_bfloat16;
    return RESBM_DISPATCH(d.dtype,
        dec_bwd_t<float>(d, (const float *)dY, (const float *)B, (const float *)Wd1,
                         (const float *)Wd2, (float *)dB, dWd1, dWd2, ws, c),
        dec_bwd_t<bf>(d, (const bf *)dY, (const bf *)B, (const bf *)Wd1, (const bf *)Wd2,
                      (bf *)dB, dWd1, dWd2, ws, c));
}

cudaError_t generic_encode_bwd(const resbm_desc &d, const void *dB, const void *F,
                               const float *P_save, const void *We1, const void *We2, void *dF,
                               void *dX, float *dWe1, float *dWe2, void *ws, const Ctx &c)
{
    using bf = __nv_bfloat16;
    return RESBM_DISPATCH(d.dtype,
        enc_bwd_t<float>(d, (const float *)dB, (const float *)F, P_save, (const float *)We1,
                         (const float *)We2, (float *)dF, (float *)dX, dWe1, dWe2, ws, c),
        enc_bwd_t<bf>(d, (const bf *)dB, (const bf *)F, P_save, (const bf *)We1,
                      (const bf *)We2, (bf *)dF, (bf *)dX, dWe1, dWe2, ws, c));
}

cudaError_t fill_identity(const resbm_desc &d, void *out, const Ctx &c)
{
    const int64_t n = d.r;
    if (d.dtype == RESBM_F32)
        k_identity<float><<<grid_for(n * n, c), 256, 0, c.stream>>>(static_cast<float *>(out), n);
    else
        k_identity<__nv_bfloat16><<<grid_for(n * n, c), 256, 0, c.stream>>>(static_cast<__nv_bfloat16 *>(out), n);
    count_launches(1);
    return cudaGetLastError();
}

}  // namespace resbm
