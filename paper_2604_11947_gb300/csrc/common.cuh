// common.cuh -- device helpers shared by the ResBM boundary kernels.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "resbm.h"

namespace resbm {

// ---- element conversion ------------------------------------------------------------------
__device__ __forceinline__ float to_f32(float v) { return v; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 v) { return __bfloat162float(v); }

template <typename T> __device__ __forceinline__ T from_f32(float v);
template <> __device__ __forceinline__ float from_f32<float>(float v) { return v; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float v)
{
    return __float2bfloat16_rn(v);
}

// ---- the nonlinearity phi of Sec. 3.2 and its derivative -----------------------------------
// SiLU(x) = x * sigmoid(x);  SiLU'(x) = s + x s (1 - s).
// GELU(x) = 0.5 x (1 + tanh(u)), u = sqrt(2/pi) (x + 0.044715 x^3);
// GELU'(x) = 0.5 (1 + tanh u) + 0.5 x (1 - tanh^2 u) sqrt(2/pi) (1 + 3 * 0.044715 x^2).
constexpr float kSqrt2OverPi = 0.7978845608028654f;
constexpr float kGeluC = 0.044715f;

__device__ __forceinline__ float act_f(int act, float x)
{
    if (act == RESBM_ACT_SILU) return x / (1.0f + expf(-x));
    if (act == RESBM_ACT_GELU_TANH) {
        const float u = kSqrt2OverPi * fmaf(kGeluC * x, x * x, x);
        return 0.5f * x * (1.0f + tanhf(u));
    }
    return x;
}

__device__ __forceinline__ float dact_f(int act, float x)
{
    if (act == RESBM_ACT_SILU) {
        const float s = 1.0f / (1.0f + expf(-x));
        return s * fmaf(x, 1.0f - s, 1.0f);
    }
    if (act == RESBM_ACT_GELU_TANH) {
        const float u = kSqrt2OverPi * fmaf(kGeluC * x, x * x, x);
        const float th = tanhf(u);
        const float du = kSqrt2OverPi * fmaf(3.0f * kGeluC * x, x, 1.0f);
        return 0.5f * (1.0f + th) + 0.5f * x * (1.0f - th * th) * du;
    }
    return 1.0f;
}

// The same functions with CUDA's fast intrinsics (__expf, __fdividef, __tanhf-free tanh via
// __expf): used where the result feeds a bf16 tensor-core operand (rounded to 8 significant bits,
// far coarser than the intrinsics' error).
__device__ __forceinline__ float fast_tanh(float u)
{
    // tanh(u) = 1 - 2 / (exp(2u) + 1), saturating cleanly for large |u|
    return 1.0f - __fdividef(2.0f, __expf(2.0f * u) + 1.0f);
}

__device__ __forceinline__ float act_fast(int act, float x)
{
    if (act == RESBM_ACT_SILU) return __fdividef(x, 1.0f + __expf(-x));
    if (act == RESBM_ACT_GELU_TANH) {
        const float u = kSqrt2OverPi * fmaf(kGeluC * x, x * x, x);
        return 0.5f * x * (1.0f + fast_tanh(u));
    }
    return x;
}

__device__ __forceinline__ float dact_fast(int act, float x)
{
    if (act == RESBM_ACT_SILU) {
        const float s = __fdividef(1.0f, 1.0f + __expf(-x));
        return s * fmaf(x, 1.0f - s, 1.0f);
    }
    if (act == RESBM_ACT_GELU_TANH) {
        const float u = kSqrt2OverPi * fmaf(kGeluC * x, x * x, x);
        const float th = fast_tanh(u);
        const float du = kSqrt2OverPi * fmaf(3.0f * kGeluC * x, x, 1.0f);
        return 0.5f * (1.0f + th) + 0.5f * x * (1.0f - th * th) * du;
    }
    return 1.0f;
}

// act and its derivative at the same point (one exp / tanh)
__device__ __forceinline__ void act_and_dact(int act, float x, float &a, float &da)
{
    if (act == RESBM_ACT_SILU) {
        const float s = 1.0f / (1.0f + expf(-x));
        a = x * s;
        da = s * fmaf(x, 1.0f - s, 1.0f);
    } else if (act == RESBM_ACT_GELU_TANH) {
        const float u = kSqrt2OverPi * fmaf(kGeluC * x, x * x, x);
        const float th = tanhf(u);
        const float du = kSqrt2OverPi * fmaf(3.0f * kGeluC * x, x, 1.0f);
        a = 0.5f * x * (1.0f + th);
        da = 0.5f * (1.0f + th) + 0.5f * x * (1.0f - th * th) * du;
    } else {
        a = x;
        da = 1.0f;
    }
}

// ---- the same functions over a row of N values -----------------------------------------------
// The branch on the activation is taken once, outside the element loop, so that the N
// independent evaluations interleave instead of running one after the other.
#define RESBM_ACT_ROW_LOOP(ACT, BODY)                                                 \
    do {                                                                              \
        if ((ACT) == RESBM_ACT_SILU) {                                                \
            constexpr int kAct = RESBM_ACT_SILU;                                      \
            _Pragma("unroll") for (int j = 0; j < N; ++j) { BODY; }                   \
        } else if ((ACT) == RESBM_ACT_GELU_TANH) {                                    \
            constexpr int kAct = RESBM_ACT_GELU_TANH;                                 \
            _Pragma("unroll") for (int j = 0; j < N; ++j) { BODY; }                   \
        } else {                                                                      \
            constexpr int kAct = RESBM_ACT_IDENTITY;                                  \
            _Pragma("unroll") for (int j = 0; j < N; ++j) { BODY; }                   \
        }                                                                             \
    } while (0)

// v = phi(v), precise or fast
template <int N> __device__ __forceinline__ void act_row(int act, float (&v)[N])
{
    RESBM_ACT_ROW_LOOP(act, v[j] = act_f(kAct, v[j]));
}
template <int N> __device__ __forceinline__ void act_fast_row(int act, float (&v)[N])
{
    RESBM_ACT_ROW_LOOP(act, v[j] = act_fast(kAct, v[j]));
}
// d = phi'(x), fast (d may alias x)
template <int N> __device__ __forceinline__ void dact_fast_row(int act, const float (&x)[N], float (&d)[N])
{
    RESBM_ACT_ROW_LOOP(act, d[j] = dact_fast(kAct, x[j]));
}
// a = phi(x), d = phi'(x), precise
template <int N> __device__ __forceinline__ void act_dact_row(int act, const float (&x)[N], float (&a)[N], float (&d)[N])
{
    RESBM_ACT_ROW_LOOP(act, act_and_dact(kAct, x[j], a[j], d[j]));
}
// a = phi(x), d = phi'(x), fast
template <int N> __device__ __forceinline__ void act_dact_fast_row(int act, const float (&x)[N], float (&a)[N], float (&d)[N])
{
    RESBM_ACT_ROW_LOOP(act, (a[j] = act_fast(kAct, x[j]), d[j] = dact_fast(kAct, x[j])));
}

}  // namespace resbm
