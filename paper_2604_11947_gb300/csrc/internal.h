// internal.h -- host-side interfaces between the C ABI layer and the kernel files.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "resbm.h"

namespace resbm {

// Counts every kernel this library enqueues (resbm_kernel_launches()).
void count_launches(uint64_t n);

struct Ctx {
    cudaStream_t stream;
    int device;
    int sm_count;
};

// Bump-allocates 256-byte aligned regions out of the caller's workspace (or, with a null
// base, only measures them).
struct WsCarver {
    char *base;
    size_t used = 0;
    explicit WsCarver(void *b) : base(static_cast<char *>(b)) {}
    template <typename T> T *take(size_t count)
    {
        used = (used + 255) & ~size_t(255);
        T *p = base ? reinterpret_cast<T *>(base + used) : nullptr;
        used += count * sizeof(T);
        return p;
    }
};

// ---- generic CUDA-core path (any shape, fp32 or bf16) ------------------------------------
size_t generic_ws_bytes(const resbm_desc &d, int op);
// out (r x r, the descriptor's dtype) = the identity matrix
cudaError_t fill_identity(const resbm_desc &d, void *out, const Ctx &c);
cudaError_t generic_encode_fwd(const resbm_desc &d, const void *X, const void *F, const void *We1,
                               const void *We2, void *B, float *P_save, void *ws, const Ctx &c);
cudaError_t generic_decode_fwd(const resbm_desc &d, const void *B, const void *Wd1,
                               const void *Wd2, void *Y, void *ws, const Ctx &c);
cudaError_t generic_decode_bwd(const resbm_desc &d, const void *dY, const void *B,
                               const void *Wd1, const void *Wd2, void *dB, float *dWd1,
                               float *dWd2, void *ws, const Ctx &c);
cudaError_t generic_encode_bwd(const resbm_desc &d, const void *dB, const void *F,
                               const float *P_save, const void *We1, const void *We2, void *dF,
                               void *dX, float *dWe1, float *dWe2, void *ws, const Ctx &c);
// Backward of N = RMSNorm(Y) * gamma with an incoming dY added (dY may be null or equal dY_out):
// dY_out (T x d, the descriptor's dtype) and dgamma (d, fp32). ws: rmsnorm_bwd_ws_bytes(d).
bool rmsnorm_bwd_supported(const resbm_desc &d);
size_t rmsnorm_bwd_ws_bytes(const resbm_desc &d);
cudaError_t generic_rmsnorm_bwd(const resbm_desc &d, const void *Y, const void *gamma, float eps, const void *dN,
                                const void *dY, void *dY_out, float *dgamma, void *ws, const Ctx &c);
// N = RMSNorm(Y) * gamma over rows of d (the descriptor's dtype), reading a stored Y
cudaError_t generic_rmsnorm(const resbm_desc &d, const void *Y, const void *gamma, float eps, void *N,
                            const Ctx &c);

}  // namespace resbm
