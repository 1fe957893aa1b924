// tc_spectral.cuh -- small kernels of the two matrix utilities around the bottleneck weights
// (Sec. 3.4.2 and the appendix's spectral analysis): the Frobenius normalisation that starts
// Muon's Newton-Schulz orthogonalisation, and the top eigenvalue of a Gram matrix W^T W by power
// iteration for the effective rank r_eff = sum sigma_i^2 / max sigma_i^2 = trace(W^T W) /
// lambda_max(W^T W). The products themselves run on the tensor-core GEMM (tc_gemm.cuh).
// Every sum here has a fixed order (per-block ranges, then the blocks in order): results are
// bitwise reproducible.
#pragma once

#include "common.cuh"
#include "tc_common.cuh"

namespace resbm {
namespace tc {

constexpr int kSqBlocks = 256;   // blocks of the sum-of-squares pass (fixed: a fixed summation order)

template <typename T> __device__ __forceinline__ float ld_f(const T *p, int64_t i) { return to_f32(p[i]); }

// part[b] = sum of x[i]^2 over block b's contiguous range (fp64), b < gridDim.x = kSqBlocks
template <typename T>
__global__ void __launch_bounds__(256) k_sumsq(const T *__restrict__ x, int64_t n, double *__restrict__ part)
{
    __shared__ double red[256];
    griddep_wait();
    griddep_launch_dependents();
    const int64_t per = (n + gridDim.x - 1) / gridDim.x;
    const int64_t b0 = blockIdx.x * per, b1 = b0 + per < n ? b0 + per : n;
    double s = 0.0;
    for (int64_t i = b0 + threadIdx.x; i < b1; i += blockDim.x) {
        const double v = ld_f(x, i);
        s = fma(v, v, s);
    }
    red[threadIdx.x] = s;
    __syncthreads();
    for (int w = 128; w > 0; w >>= 1) {
        if ((int)threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
        __syncthreads();
    }
    if (threadIdx.x == 0) part[blockIdx.x] = red[0];
}

// y = bf16(x / (||x||_F + eps)), ||x||_F^2 the sum of the kSqBlocks partials in block order
template <typename T>
__global__ void __launch_bounds__(256) k_scale_bf16(const T *__restrict__ x, int64_t n, const double *__restrict__ part,
                                                    float eps, __nv_bfloat16 *__restrict__ y)
{
    griddep_wait();
    griddep_launch_dependents();
    double s = 0.0;
    for (int b = 0; b < kSqBlocks; ++b) s += part[b];
    const float inv = (float)(1.0 / (sqrt(s) + (double)eps));
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        y[i] = __float2bfloat16_rn(ld_f(x, i) * inv);
}

// Power iteration on a symmetric positive semi-definite n x n fp32 matrix G (row-major) by one
// CTA: v <- G v / ||G v|| from a fixed start vector, until the residual ||G v - lambda v|| of the
// Rayleigh quotient lambda = v^T G v (||v|| = 1) is at most tol * lambda, or max_iter iterations.
// For a symmetric matrix some eigenvalue lies within the residual of lambda (Bauer-Fike), so the
// stop bounds the eigenvalue's relative error by tol even when the top eigenvalues are close
// (where the Rayleigh quotient itself creeps slowly). out[0] = lambda_max,
// out[1] = trace(G) (fp64 sum in index order), out[2] = trace / lambda_max (the effective rank
// when G = W^T W), out[3] = iterations taken. The vectors live in shared memory (n <= kPowMaxN).
constexpr int kPowMaxN = 4096;
__global__ void __launch_bounds__(1024) k_power_iter(const float *__restrict__ G, int n, int max_iter, float tol,
                                                     double *__restrict__ out)
{
    __shared__ float v[kPowMaxN], y[kPowMaxN];
    __shared__ double red[32];
    __shared__ double bc;
    griddep_wait();
    griddep_launch_dependents();
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nw = blockDim.x >> 5;
    // a fixed start with no special direction: 1 + 0.5 sin(0.7 j)
    for (int j = tid; j < n; j += blockDim.x) v[j] = 1.0f + 0.5f * sinf(0.7f * (float)j);
    __syncthreads();
    // block-wide sum of per-thread doubles in a fixed order
    auto block_sum = [&](double t) -> double {
        for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
        if (lane == 0) red[warp] = t;
        __syncthreads();
        if (tid == 0) {
            double s = 0.0;
            for (int w = 0; w < nw; ++w) s += red[w];
            bc = s;
        }
        __syncthreads();
        const double r = bc;
        __syncthreads();
        return r;
    };
    double nv = 0.0;
    for (int j = tid; j < n; j += blockDim.x) nv += (double)v[j] * v[j];
    nv = block_sum(nv);
    const float s0 = (float)(1.0 / sqrt(nv));
    for (int j = tid; j < n; j += blockDim.x) v[j] *= s0;
    __syncthreads();
    double lam = 0.0;
    int it = 0;
    for (; it < max_iter; ++it) {
        // y = G v: one warp per row, lanes along the row, a fixed reduction tree
        for (int i = warp; i < n; i += nw) {
            float acc = 0.0f;
            for (int j = lane; j < n; j += 32) acc = fmaf(G[(int64_t)i * n + j], v[j], acc);
            for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
            if (lane == 0) y[i] = acc;
        }
        __syncthreads();
        double rq = 0.0, ny = 0.0, vv = 0.0;
        for (int j = tid; j < n; j += blockDim.x) {
            rq += (double)v[j] * y[j];
            ny += (double)y[j] * y[j];
            vv += (double)v[j] * v[j];
        }
        rq = block_sum(rq);
        ny = block_sum(ny);
        vv = block_sum(vv);
        lam = rq / vv;   // the Rayleigh quotient of v (unit length up to fp32 rounding)
        if (ny <= 0.0) break;   // G v = 0: G is zero on the start vector's span
        // the residual ||G v - lam v|| / ||v||, summed element by element in fp64
        double r2 = 0.0;
        for (int j = tid; j < n; j += blockDim.x) {
            const double t = (double)y[j] - lam * (double)v[j];
            r2 += t * t;
        }
        const double res = sqrt(block_sum(r2) / vv);
        const float s = (float)(1.0 / sqrt(ny));
        for (int j = tid; j < n; j += blockDim.x) v[j] = y[j] * s;
        __syncthreads();
        if (res <= (double)tol * fabs(lam)) {
            ++it;
            break;
        }
    }
    if (tid == 0) {
        double tr = 0.0;
        for (int i = 0; i < n; ++i) tr += (double)G[(int64_t)i * n + i];
        out[0] = lam;
        out[1] = tr;
        out[2] = lam > 0.0 ? tr / lam : 0.0;
        out[3] = (double)it;
    }
}

}  // namespace tc
}  // namespace resbm
