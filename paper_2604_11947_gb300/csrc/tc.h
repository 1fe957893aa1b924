// tc.h -- host-side interface of the sm_103a tensor-core (tcgen05 + TMA) kernels.
#pragma once

#include "internal.h"

namespace resbm {

// Whether the tensor-core kernels handle this descriptor for `op` (bf16 I/O, shapes that fit
// their tiles); otherwise the portable kernels run.
bool tc_supported(const resbm_desc &d, int op);

// Reads (and optionally clears) the error word of the tensor-core kernels; synchronizing.
cudaError_t tc_device_error(unsigned int *code, bool clear);
// Enqueues a one-CTA kernel whose only wait can never complete: it gives up after the bounded
// wait time and records the timeout in the error word (a test of that path; nothing faults).
cudaError_t tc_wait_selftest(const Ctx &c);
// One launch of the HBM access-form probe `form` (resbm_hbm_form, tc_hbm_forms.cuh) over `bytes`
// bytes: a is read, b written (arguments checked by the caller).
cudaError_t tc_hbm_form(int form, const void *a, void *b, int64_t bytes, const Ctx &c);
// Scratch bytes of the tensor-core kernels for `op` on a device with `sms` SMs.
size_t tc_ws_bytes(const resbm_desc &d, int op, int sms);

cudaError_t tc_encode_fwd(const resbm_desc &d, const void *X, const void *F, const void *We1,
                          const void *We2, void *B, float *P_save, void *ws, const Ctx &c);
cudaError_t tc_decode_fwd(const resbm_desc &d, const void *B, const void *Wd1, const void *Wd2,
                          void *Y, void *ws, const Ctx &c);
// The decoder forward with the next block's pre-attention RMSNorm fused in (k_dec_fwd's NORM
// passes): Y and N = Y / sqrt(mean_j Y_j^2 + eps) * gamma. ws: tc_rmsnorm_ws_bytes(d) bytes (the
// row sums of squares), 16-byte aligned.
size_t tc_rmsnorm_ws_bytes(const resbm_desc &d);
cudaError_t tc_decode_fwd_rmsnorm(const resbm_desc &d, const void *B, const void *Wd1, const void *Wd2,
                                  const void *gamma, float eps, void *Y, void *N, void *ws, const Ctx &c);
// after_independent: the previous kernel on c.stream is the boundary step's decoder forward of
// the same B (it reads B and writes Y only, and B was complete before it could let this launch
// begin), so the kernel starts on SMs as that kernel's CTAs leave, without waiting for its end
// (it waits for it before it exits, so it never completes first: later kernels of the stream,
// which wait for their predecessor only, still find the decoder forward complete).
cudaError_t tc_decode_bwd(const resbm_desc &d, const void *dY, const void *B, const void *Wd1,
                          const void *Wd2, void *dB, float *dWd1, float *dWd2, void *ws,
                          const Ctx &c, bool after_independent = false);
cudaError_t tc_encode_bwd(const resbm_desc &d, const void *dB, const void *F, const float *P_save,
                          const void *We1, const void *We2, void *dF, void *dX, float *dWe1,
                          float *dWe2, void *ws, const Ctx &c);

// The GEMM chain (tc_gemm.cuh): every op as a sequence of tcgen05 products with fused
// epilogues, for bf16 shapes the fused kernels do not take (m = r = 512, the r = 128 backward,
// m != r). Needs d, r, m multiples of 8 and 16-byte aligned pointers (else cudaErrorNotSupported
// before anything is enqueued).
bool gemm_supported(const resbm_desc &d, int op);
size_t gemm_ws_bytes(const resbm_desc &d, int op, int sms);
cudaError_t gemm_encode_fwd(const resbm_desc &d, const void *X, const void *F, const void *We1,
                            const void *We2, void *B, float *P_save, void *ws, const Ctx &c);
cudaError_t gemm_decode_fwd(const resbm_desc &d, const void *B, const void *Wd1, const void *Wd2,
                            void *Y, void *ws, const Ctx &c);
cudaError_t gemm_decode_bwd(const resbm_desc &d, const void *dY, const void *B, const void *Wd1,
                            const void *Wd2, void *dB, float *dWd1, float *dWd2, void *ws,
                            const Ctx &c);
cudaError_t gemm_encode_bwd(const resbm_desc &d, const void *dB, const void *F, const float *P_save,
                            const void *We1, const void *We2, void *dF, void *dX, float *dWe1,
                            float *dWe2, void *ws, const Ctx &c);

// Muon's Newton-Schulz orthogonalisation and the effective rank of a matrix (tc_spectral.cuh and
// the GEMM): rows, cols multiples of 8; 16-byte aligned pointers (else cudaErrorNotSupported
// before anything is enqueued).
bool matrix_supported(int64_t rows, int64_t cols);
size_t matrix_ws_bytes(int op, int64_t rows, int64_t cols, int sms);
cudaError_t tc_newton_schulz(int64_t rows, int64_t cols, const void *G, bool g_f32, int steps,
                             const float coef[3], float eps, void *X_out, void *ws, const Ctx &c);
cudaError_t tc_effective_rank(int64_t rows, int64_t cols, const void *W, double *out, void *ws,
                              const Ctx &c);

// The encoder fused into the FFN down-projection (tc_gemm.cuh, ENCP): F = H . W2 on the tensor
// cores, P = F . We1 accumulated from the F tiles in the epilogue into per-tile partial slots, then
// B = X[:, :r] + phi(P) . We2; F reaches memory only when F_out is set. bf16, m % 8 == 0, m, r <= 32.
bool ffn_encode_supported(const resbm_desc &d, int64_t f);
size_t ffn_encode_ws_bytes(const resbm_desc &d, int64_t f);
cudaError_t tc_ffn_down_encode(const resbm_desc &d, int64_t f, const void *H, const void *W2, const void *X,
                               const void *We1, const void *We2, void *B, float *P, void *F_out, void *ws,
                               const Ctx &c);

}  // namespace resbm
