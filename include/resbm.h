/*
 * resbm.h -- C ABI of the ResBM boundary bottleneck on one GB300 (sm_103a).
 *
 * ResBM (Residual Bottleneck Models, arXiv 2604.11947) places an autoencoder across every
 * pipeline-stage boundary (Sec. 3.2): the encoder E at the end of block l compresses the
 * feed-forward output z_l (T x d) to the boundary tensor b_l (T x r, r < d), which is the only
 * tensor that crosses the boundary; the decoder D at the start of block l+1 expands it back
 * to T x d. Both are "two linear layers with a non-linearity applied between them" (Sec. 3.2).
 * The identity path survives the change of width through the fixed projection
 * P^id(x) = x . I_{c x C} (Eq. rect_identity_definition, Eq. Pid_definition): truncation to
 * the first r columns on the sending side, zero padding on the receiving side, merged by the
 * generalized residual update x_{l+1} = x_l P^id + F(x_l) (Eq. generalized_transformer_equation).
 *
 * Notation (paper -> this header): L*batch -> T tokens, H -> d, h -> r, x_l^Attn -> X,
 * z_l -> F, b_l -> B; m is the hidden width between the two linear layers (the paper does not
 * fix it; m = r in the shipped workloads). All matrices are dense, row-major, in the paper's
 * "x . W" orientation:
 *     X, F, Y, dY, dF, dX : T x d        B, dB : T x r        P : T x m (fp32)
 *     We1 : d x m    We2 : m x r    Wd1 : r x m    Wd2 : m x d
 *
 * Computed (phi = the activation chosen in the descriptor):
 *   encode fwd   B  = X . I_{d x r} + phi(F . We1) . We2             P = F . We1 (saved, fp32)
 *   decode fwd   Y  = [merge] B . I_{r x d} + phi(B . Wd1) . Wd2
 *   decode bwd   dB = [merge] dY . I_{r x d}^T + ((dY . Wd2^T) * phi'(Q)) . Wd1^T,  Q = B . Wd1
 *                dWd2 = phi(Q)^T . dY        dWd1 = B^T . ((dY . Wd2^T) * phi'(Q))
 *   encode bwd   dP = (dB . We2^T) * phi'(P);  dF = dP . We1^T;  dX[:, :r] += dB
 *                dWe1 = F^T . dP            dWe2 = phi(P)^T . dB
 *
 * Conventions shared by every entry point:
 *   - Every tensor pointer is DEVICE memory owned by the caller (for example a torch tensor's
 *     storage). The library allocates nothing, frees nothing and never synchronizes: work is
 *     enqueued on `stream` (a cudaStream_t; NULL is the legacy default stream) and the call
 *     returns. Inputs must stay alive and unmodified until the enqueued work has finished.
 *   - I/O tensors and weights have the descriptor's dtype (fp32 or bf16); P and every weight
 *     gradient are fp32. Arithmetic accumulates in fp32. For bf16 the intermediates that feed a
 *     tensor-core product are rounded to bf16; outputs are rounded once, to nearest even.
 *   - Weight gradients are OVERWRITTEN (they are complete sums over the T tokens). dX is
 *     ACCUMULATED: dB is added into its first r columns and its other columns are not touched.
 *   - Arguments are validated before anything is enqueued; a failure returns a status code and
 *     enqueues nothing. The library never aborts or exits. A CUDA error at launch time returns
 *     RESBM_ERR_CUDA (resbm_last_cuda_error() gives the cudaError_t value).
 *   - Outputs must not overlap inputs (X may alias F: both are only read).
 *   - Results are deterministic: the same inputs, descriptor and device give the same bits.
 *     (The tensor-core backward kernels run in thread-block clusters of 1, 2 or 4 CTAs and the
 *     encoder forward in pairs, chosen from the device's occupancy and T; the environment
 *     variable RESBM_CLUSTER=1, 2 or 4 forces the backward size where it fits, and 1 also runs
 *     the encoder forward as single CTAs. Each choice is deterministic; different choices add in
 *     different fixed orders, so results may differ between them in the last bits.)
 *   - T = 0 is valid: nothing is read, weight gradients are set to zero.
 *   - The scratch memory `ws` (device, >= resbm_workspace_bytes(...) bytes, 256-byte aligned)
 *     belongs to the call until its work finishes; its contents on entry do not matter.
 */
#ifndef RESBM_H
#define RESBM_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define RESBM_API __attribute__((visibility("default")))
#else
#define RESBM_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    RESBM_OK = 0,
    RESBM_ERR_INVALID_ARG = 1,   /* null/misaligned pointer, bad size or enum, overlap */
    RESBM_ERR_UNSUPPORTED = 2,   /* valid request the library does not run */
    RESBM_ERR_WORKSPACE = 3,     /* ws is NULL or smaller than resbm_workspace_bytes() */
    RESBM_ERR_CUDA = 4           /* a CUDA runtime call or launch failed */
} resbm_status;

typedef enum { RESBM_F32 = 0, RESBM_BF16 = 1 } resbm_dtype;

/* phi of Sec. 3.2 (the paper does not name it): SiLU x*sigmoid(x) (default),
 * GELU tanh form 0.5x(1+tanh(sqrt(2/pi)(x+0.044715x^3))), or identity. */
typedef enum { RESBM_ACT_SILU = 0, RESBM_ACT_GELU_TANH = 1, RESBM_ACT_IDENTITY = 2 } resbm_act;

typedef enum {
    RESBM_OP_ENCODE_FWD = 0,
    RESBM_OP_DECODE_FWD = 1,
    RESBM_OP_DECODE_BWD = 2,
    RESBM_OP_ENCODE_BWD = 3,
    RESBM_OP_BOUNDARY_STEP = 4,
    RESBM_OP_BOUNDARY_STEP_HOST = 5,
    RESBM_OP_EFFECTIVE_RANK = 6,     /* resbm_effective_rank (workspace: resbm_matrix_workspace_bytes) */
    RESBM_OP_NEWTON_SCHULZ = 7,      /* resbm_newton_schulz  (workspace: resbm_matrix_workspace_bytes) */
    RESBM_OP_DECODE_FWD_RMSNORM = 8, /* resbm_decode_fwd_rmsnorm */
    RESBM_OP_RMSNORM_BWD = 9         /* resbm_rmsnorm_bwd */
} resbm_op;

/* desc.flags bits */
#define RESBM_FLAG_GENERIC 1u   /* force the portable CUDA-core kernels (no tensor cores) */
/* One linear layer on each side instead of two (the single-matrix special case of Sec. 3.2's
 * encoder / decoder): E(F) = F . We1 with We1 d x r, D(B) = B . Wd2 with Wd2 r x d. Requires
 * m == r; act is not used; We2 and Wd1 are not read and dWe2 and dWd1 not written (all may be
 * NULL). Everything else, the identity path included, is as in the two-layer form. */
#define RESBM_FLAG_LINEAR 2u
/* Run every op as its chain of tensor-core products with fused element-wise steps (the path
 * the library takes by itself for bf16 shapes the fused boundary kernels do not cover, e.g.
 * m = r = 512, or the backward at m = 128, or m != r) even where the fused kernels would run.
 * bf16 only, d, r and m multiples of 8, 16-byte aligned pointers; otherwise the portable
 * kernels run. For testing and comparing the two tensor-core paths. */
#define RESBM_FLAG_GEMM 4u

typedef struct {
    int64_t T;               /* tokens (batch * sequence), >= 0                              */
    int64_t d;               /* residual width H, >= 1                                       */
    int64_t r;               /* bottleneck width h, 1 <= r <= d (compression d / r)          */
    int64_t m;               /* hidden width of the two-layer encoder / decoder, >= 1        */
    int32_t dtype;           /* resbm_dtype of X, F, B, Y, dY, dB, dF, dX and the weights    */
    int32_t act;             /* resbm_act                                                     */
    int32_t merge_identity;  /* 1: Y = B . I_{r x d} + D(B);  0: Y = D(B) (the caller adds the
                                padded skip itself, e.g. after attention)                     */
    uint32_t flags;          /* RESBM_FLAG_* bits, 0 for the default kernels                 */
} resbm_desc;

/* Pointers for resbm_boundary_step (all device memory, layouts as above). */
typedef struct {
    const void *X, *F, *dY;                 /* inputs, T x d                                  */
    const void *We1, *We2, *Wd1, *Wd2;      /* weights                                        */
    void *B;                                /* out: T x r boundary tensor                     */
    float *P;                               /* out: T x m fp32 F.We1, or NULL (kept in ws)    */
    void *Y;                                /* out: T x d decoder output                      */
    void *dB;                               /* out: T x r gradient sent back                  */
    void *dF;                               /* out: T x d                                     */
    void *dX;                               /* in/out: T x d, first r columns += dB; or NULL  */
    float *dWe1, *dWe2, *dWd1, *dWd2;       /* out: fp32 weight gradients                     */
    /* resbm_boundary_step_host only (ignored by resbm_boundary_step; NULL for none): CUDA event
     * handles (cudaEvent_t) that chain the host-link phases of consecutive calls */
    void *wait_before_inputs;               /* the call's host-to-device copies wait for it   */
    void *inputs_done;                      /* recorded when all its host-to-device copies are done */
} resbm_step_args;

/* Library version string, e.g. "resbm 0.1.0 sm_103a". */
RESBM_API const char *resbm_version(void);

/* Human-readable name of a status code (static storage). */
RESBM_API const char *resbm_status_string(resbm_status status);

/* The cudaError_t value behind the last RESBM_ERR_CUDA returned on this host thread (0 if none). */
RESBM_API int resbm_last_cuda_error(void);

/* Number of kernels this library has enqueued in this process so far (all devices, all host
 * threads): lets a caller account for the GPU work behind a sequence of calls. */
RESBM_API uint64_t resbm_kernel_launches(void);

/* Error word of the tensor-core kernels on the current device (0: none). Every wait inside
 * those kernels gives up after a bounded time instead of spinning forever; a kernel that gave
 * up sets a bit here (1: a wait timed out; 4: a CTA's token share did not fit the launch's
 * tile-group plan, an internal error) and returns, leaving its outputs undefined.
 * Reading the word synchronizes with the device (it is a device-to-host copy). With clear != 0
 * a non-zero word is reset to 0. */
RESBM_API resbm_status resbm_device_error(unsigned int *code, int clear);

/* Failure-path self-test (no counterpart in the paper): enqueues on `stream` a one-CTA kernel
 * whose only wait can never complete. Like every wait in the tensor-core kernels it gives up
 * after its bounded time (about 2 s), sets bit 1 of the error word read by resbm_device_error()
 * and returns; nothing faults and the context stays usable. Lets a caller (and the tests) check
 * that a stuck wait is reported instead of hanging the device. */
RESBM_API resbm_status resbm_selftest_wait_timeout(void *stream);

/* Memory-system probe (no counterpart in the paper): the access forms whose HBM rates the
 * kernels' choice of load and store forms rests on. One call enqueues on `stream` one launch of
 * `form` over `bytes` bytes:
 *   RESBM_HBM_READ_V4         reads a: 16-byte loads by every thread (four 512-thread CTAs per SM)
 *   RESBM_HBM_WRITE_V4        writes b the same way (every byte 0xA5)
 *   RESBM_HBM_COPY_V4         copies a to b the same way (moves 2 * bytes)
 *   RESBM_HBM_READ_TMA_2D     reads a with one CTA per SM: 2-D tensor loads of 64-column x
 *                             128-row bf16 boxes (16 KB, 128-byte swizzle), 8 stages in flight
 *   RESBM_HBM_READ_TMA_2D_PAIR two such boxes per 32 KB stage on one barrier, 4 stages
 *   RESBM_HBM_READ_TMA_3D     one 3-D box of two neighbouring 64-column blocks per 32 KB stage
 *   RESBM_HBM_READ_BULK       1-D bulk copies of 16 KB, 8 stages
 *   RESBM_HBM_WRITE_TMA_2D    writes b with 2-D tensor stores of the 64 x 128 boxes (0xA5)
 *   RESBM_HBM_WRITE_BULK      writes b with 1-D bulk stores of 16 KB (0xA5)
 *   RESBM_HBM_READ_TMA_2D_TILES  as RESBM_HBM_READ_TMA_2D_PAIR in the backward kernels' walk:
 *                             each CTA's run of 128-row tiles in groups of up to four, per group
 *                             the 128-column chunks in cyclic order from a chunk that depends on
 *                             the CTA, each chunk's tiles one after the other
 *   RESBM_HBM_WRITE_TMA_2D_TILES  as RESBM_HBM_WRITE_TMA_2D in that walk (0xA5)
 * The TMA forms view a buffer as a row-major bf16 matrix of 4096 columns (8 KB rows); each
 * CTA streams a contiguous run of its boxes (row-tile-major unless a form says otherwise). a and b: device memory of `bytes` bytes each,
 * 16-byte aligned, not overlapping, both required for every form (RESBM_HBM_READ_V4 writes at
 * most 4 bytes of b, and only for an input it does not expect). bytes: a positive multiple of
 * 1 MiB. Errors: RESBM_ERR_INVALID_ARG for a bad form, size or pointer (nothing enqueued);
 * RESBM_ERR_CUDA if a launch (or the tensor-map encoding) failed. Waits are bounded as in the
 * other tensor-core kernels (resbm_device_error reports a timeout). */
typedef enum {
    RESBM_HBM_READ_V4 = 0,
    RESBM_HBM_WRITE_V4 = 1,
    RESBM_HBM_COPY_V4 = 2,
    RESBM_HBM_READ_TMA_2D = 3,
    RESBM_HBM_READ_TMA_2D_PAIR = 4,
    RESBM_HBM_READ_TMA_3D = 5,
    RESBM_HBM_READ_BULK = 6,
    RESBM_HBM_WRITE_TMA_2D = 7,
    RESBM_HBM_WRITE_BULK = 8,
    RESBM_HBM_READ_TMA_2D_TILES = 9,
    RESBM_HBM_WRITE_TMA_2D_TILES = 10
} resbm_hbm_form;
RESBM_API resbm_status resbm_measure_hbm_form(int form, const void *a, void *b, int64_t bytes, void *stream);

/* Scratch bytes that `op` (a resbm_op) needs for `desc`, written to *bytes.
 * Returns RESBM_ERR_INVALID_ARG for a bad descriptor or op. Does not touch the GPU. */
RESBM_API resbm_status resbm_workspace_bytes(const resbm_desc *desc, int op, size_t *bytes);

/* Send side, Sec. 3.2 (encoder at the end of block l) with the truncating identity path of
 * Eq. Pid (c = d > C = r): B = X[:, :r] + phi(F . We1) . We2.
 *   X   : T x d, only its first r columns are read (x_l^Attn, the skip source)
 *   F   : T x d (z_l, the feed-forward output); may be the same pointer as X
 *   B   : T x r out. P_save: T x m fp32 out (F . We1, reused by resbm_encode_bwd) or NULL. */
RESBM_API resbm_status resbm_encode_fwd(const resbm_desc *desc, const void *X, const void *F,
                              const void *We1, const void *We2, void *B, float *P_save,
                              void *ws, size_t ws_bytes, void *stream);

/* Receive side, Sec. 3.2 (decoder at the start of block l+1) with the zero-padding identity
 * path of Eq. Pid (c = r < C = d): Y = [merge] B . I_{r x d} + phi(B . Wd1) . Wd2.
 *   B : T x r in.  Y : T x d out. */
RESBM_API resbm_status resbm_decode_fwd(const resbm_desc *desc, const void *B, const void *Wd1,
                              const void *Wd2, void *Y, void *ws, size_t ws_bytes,
                              void *stream);

/* The receive side with the next block's pre-attention RMSNorm fused in. Sec. 3.2 places the
 * decoder at the start of block l+1, whose first step in a pre-norm transformer normalises the
 * residual stream before attention (the paper's 1B model, Sec. 4.1: RMSNorm). Returns both
 *   Y = [merge] B . I_{r x d} + phi(B . Wd1) . Wd2          (as resbm_decode_fwd; the residual stream)
 *   N[t, j] = Y[t, j] / sqrt(mean_j Y[t, j]^2 + eps) * gamma[j]   (the attention's input)
 * with the row's RMS taken over Y as stored (rounded to the descriptor's dtype). On the fused
 * tensor-core path N = round(y * rstd * gamma) with y the unrounded value of Y[t, j] (one rounding
 * fewer than normalising the stored Y: the two differ by less than half Y's spacing times
 * rstd * gamma[j] before N's rounding); elsewhere the norm reads the stored Y.
 *   gamma : d elements, the descriptor's dtype (the norm's weight); eps >= 0
 *   Y, N  : T x d out (distinct buffers)
 * On the fused tensor-core path Y is not read back from memory: the decoder runs twice, the
 * first pass storing Y and each row's partial sums of squares (fixed slots in `ws`), the second
 * recomputing the same Y bits and storing N; elsewhere the norm reads the stored Y. The row sums
 * have a fixed order, so N is bitwise reproducible. `ws`: resbm_workspace_bytes(desc,
 * RESBM_OP_DECODE_FWD_RMSNORM). Errors: as resbm_decode_fwd, and RESBM_ERR_INVALID_ARG for a null
 * gamma or N, a negative or non-finite eps, or Y and N overlapping. */
RESBM_API resbm_status resbm_decode_fwd_rmsnorm(const resbm_desc *desc, const void *B, const void *Wd1,
                                                const void *Wd2, const void *gamma, float eps, void *Y,
                                                void *N, void *ws, size_t ws_bytes, void *stream);

/* Backward of the receiving block's RMSNorm (N of resbm_decode_fwd_rmsnorm) with the residual
 * stream's own gradient added, so that resbm_decode_bwd can take the sum:
 *   dY_out = dY + dN . dN/dY,  i.e. per row  dY + s (dN * gamma) - Y (s^3 / d) sum_j dN_j gamma_j Y_j
 *   dgamma = sum_t dN[t, :] * Y[t, :] * s_t            (fp32, d)
 * with s = 1 / sqrt(mean_j Y_j^2 + eps) from Y as stored (the chain rule of the norm's three steps).
 *   Y, dN : T x d in (the descriptor's dtype); gamma: d; dY: T x d in, or NULL for zero; dY_out:
 *   T x d out, may be the same buffer as dY (in place) but not overlap Y, dN or gamma; dgamma: d
 *   fp32 out. Requires d <= 16384 (RESBM_ERR_UNSUPPORTED otherwise). Bitwise reproducible on any
 *   device (fixed row ranges and summation orders). `ws`: resbm_workspace_bytes(desc,
 *   RESBM_OP_RMSNORM_BWD) (the dgamma partials). Errors: as resbm_decode_fwd_rmsnorm. */
RESBM_API resbm_status resbm_rmsnorm_bwd(const resbm_desc *desc, const void *Y, const void *gamma, float eps,
                                         const void *dN, const void *dY, void *dY_out, float *dgamma, void *ws,
                                         size_t ws_bytes, void *stream);

/* Backward of resbm_decode_fwd for the upstream gradient dY (the compressed gradient dB is
 * what crosses the boundary backwards, Appendix A.3).
 *   dY : T x d in.  B : T x r in (the forward input).  dB : T x r out.
 *   dWd1 : r x m fp32 out.  dWd2 : m x d fp32 out. */
RESBM_API resbm_status resbm_decode_bwd(const resbm_desc *desc, const void *dY, const void *B,
                              const void *Wd1, const void *Wd2, void *dB, float *dWd1,
                              float *dWd2, void *ws, size_t ws_bytes, void *stream);

/* Backward of resbm_encode_fwd for the upstream gradient dB.
 *   dB : T x r in.  F : T x d in.  P_save : T x m fp32 from resbm_encode_fwd, or NULL
 *   (then F . We1 is recomputed, which reads F twice).
 *   dF : T x d out.  dX : T x d in/out, dX[:, :r] += dB (gradient of the truncating identity
 *   path), or NULL to skip.  dWe1 : d x m fp32 out.  dWe2 : m x r fp32 out. */
RESBM_API resbm_status resbm_encode_bwd(const resbm_desc *desc, const void *dB, const void *F,
                              const float *P_save, const void *We1, const void *We2,
                              void *dF, void *dX, float *dWe1, float *dWe2,
                              void *ws, size_t ws_bytes, void *stream);

/* Size of the library's fixed device scratch array used by resbm_decode_bwd_noalloc (32 MiB
 * per device). */
#define RESBM_STATIC_SCRATCH_BYTES ((size_t)32 << 20)

/* resbm_decode_bwd without a workspace argument: the same computation, kernels and results,
 * with its scratch taken from a fixed array that the library holds in device memory
 * (RESBM_STATIC_SCRATCH_BYTES, reserved when the library's device code is loaded) instead of
 * from the caller. The paper has no counterpart: this entry point is a library convenience.
 *
 * It is meant for callers that cannot hand over device memory for scratch: a C or C++ program
 * that links this library without a device allocator of its own, or a runtime that fixes its
 * device memory at start-up and may not allocate (or free) during a training step. Nothing is
 * allocated or freed by the call, on the device or on the host.
 *   - Arguments and results are those of resbm_decode_bwd. The scratch needed is the
 *     resbm_workspace_bytes(desc, RESBM_OP_DECODE_BWD) figure; a call that needs more than
 *     RESBM_STATIC_SCRATCH_BYTES returns RESBM_ERR_WORKSPACE and enqueues nothing. With the
 *     tensor-core kernels on 152 SMs this admits d * m up to about 55,000: d = 1024 with
 *     m = 32 fits, d = 4096 with m = 32 does not.
 *   - Nothing in the array has to start at zero: every call writes the scratch it reads.
 *   - The first call on each device looks up the array's device address (cudaGetSymbolAddress)
 *     and keeps it; make that first call on a device before starting any stream capture on it.
 *   - There is ONE array per device, shared by every call on that device. Calls enqueued on one
 *     stream run one after the other and are safe; calls whose work can overlap in time (on
 *     different streams, or from different host threads without ordering) race on the array
 *     and give undefined results. Use resbm_decode_bwd with separate workspaces for those. */
RESBM_API resbm_status resbm_decode_bwd_noalloc(const resbm_desc *desc, const void *dY,
                                      const void *B, const void *Wd1, const void *Wd2,
                                      void *dB, float *dWd1, float *dWd2, void *stream);

/* One boundary forward and backward on one GPU, the pipeline handoff kept in device memory:
 * encode_fwd -> decode_fwd -> decode_bwd -> encode_bwd, in that order on `stream`. B produced
 * by the encoder is what the decoder reads; dB produced by the decoder backward is what the
 * encoder backward reads. */
RESBM_API resbm_status resbm_boundary_step(const resbm_desc *desc, const resbm_step_args *args,
                                 void *ws, size_t ws_bytes, void *stream);

/* resbm_boundary_step with every tensor of `args` in HOST memory. The paper has no counterpart:
 * this is the host-memory form of the step, a library convenience for callers whose tensors
 * live on the host (and the form the end-to-end measurement goes through).
 *   - Same arguments, rules and results as resbm_boundary_step, except that every pointer in
 *     `args` is a host pointer. Page-locked memory (cudaHostAlloc, cudaHostRegister) lets the
 *     copies run asynchronously; with pageable memory they block the calling thread.
 *   - `ws` is DEVICE memory of resbm_workspace_bytes(desc, RESBM_OP_BOUNDARY_STEP_HOST) bytes
 *     (256-byte aligned): a device copy of every tensor of the step plus the step's own scratch.
 *   - Only what the step reads crosses to the device: X[:, :r] (the identity path is the only
 *     use of X), F, dY, the weights, and dX[:, :r] when dX is given; what comes back is B, Y, dB,
 *     dF, dX[:, :r] (dX given), P (P given) and the weight gradients. The rest of dX is not
 *     touched. When X or dX is page-locked and mapped into the device's address space (as
 *     cudaHostAlloc memory is), a small kernel reads or writes those r columns in place through
 *     the mapping; otherwise a strided copy moves them.
 *   - Everything is enqueued on `stream` (the call returns once it is enqueued; the host
 *     outputs are complete when `stream` reaches that point). Inside the call dY travels on a
 *     second stream while the forward stages run, and B and Y travel back on a third while the
 *     backward stages run; both are forked from and joined back into `stream`. Calls on
 *     different streams with different workspaces may run at the same time, so a caller can
 *     overlap one step's results with the next step's inputs.
 *   - Pipelining calls: with two calls in flight on two streams, nothing orders their copies, so
 *     both calls' inputs share the host-to-device direction at once and both results the other
 *     way. Passing call k's `inputs_done` event as call k+1's `wait_before_inputs` makes call k+1's
 *     inputs travel in while call k computes and sends its results back, one transfer per
 *     direction on the host link. Both events are optional; each call waits only on an event a
 *     call enqueued before it recorded, so the chain cannot deadlock.
 *   - The two side streams and five events are created on the first call for each (device,
 *     caller stream) pair and kept until the process exits (creating them in every call costs
 *     driver time). A caller that passes a new stream to every call therefore accumulates two
 *     streams and five events per distinct stream handle: reuse a small set of streams.
 *   - Errors: as resbm_boundary_step; RESBM_ERR_CUDA if a copy or a stream could not be set up. */
RESBM_API resbm_status resbm_boundary_step_host(const resbm_desc *desc, const resbm_step_args *args,
                                      void *ws, size_t ws_bytes, void *stream);

/* ---- the encoder fused into the feed-forward down-projection -------------------------------------
 * Sec. 3.2 places the encoder after the feed-forward layer: z = F = H . W2 (the down-projection of
 * the FFN hidden state H) is the encoder's input. This entry point computes F on the tensor cores
 * and feeds each output tile straight into the encoder (P = F . We1 accumulated from the tiles,
 * then B = X[:, :r] + phi(P) . We2), so F does not travel through memory unless asked for.
 *   H      T x f bf16 (the FFN hidden state, f = the FFN width), W2 f x d bf16
 *   X      T x d bf16 (the encoder's skip input; only its first r columns are read)
 *   We1    d x m, We2 m x r (bf16); B T x r bf16 (output); P_save T x m fp32 or NULL
 *   F_out  T x d bf16 or NULL: F itself, rounded to bf16 (what the encoder's backward reads)
 * The encoder sees F rounded to bf16, as it would if F were stored first. Requirements: bf16,
 * two linear layers (not RESBM_FLAG_LINEAR), m a multiple of 8 with m <= 32, r <= 32, d and f
 * multiples of 8, 16-byte aligned pointers; otherwise RESBM_ERR_UNSUPPORTED. `ws`: device memory of
 * resbm_ffn_down_encode_workspace_bytes(desc, f) bytes (the partial P slots), 256-byte aligned. */
RESBM_API resbm_status resbm_ffn_down_encode_workspace_bytes(const resbm_desc *desc, int64_t f, size_t *bytes);
RESBM_API resbm_status resbm_ffn_down_encode_fwd(const resbm_desc *desc, int64_t f, const void *H,
                                       const void *W2, const void *X, const void *We1,
                                       const void *We2, void *B, float *P_save, void *F_out,
                                       void *ws, size_t ws_bytes, void *stream);

/* ---- utilities on the bottleneck weights (outside the boundary op) ----------------------------
 * Two dense kernels on a bf16 matrix, for training the bottleneck weights with Muon (Sec. 3.4.2:
 * the bottleneck models are trained with Muon, whose update orthogonalises the gradient momentum
 * by a Newton-Schulz iteration) and for the appendix's spectral analysis of them (the effective
 * rank). Shapes: rows and cols multiples of 8; all pointers device memory, 16-byte aligned; `ws`
 * device memory of resbm_matrix_workspace_bytes(op, rows, cols) bytes, 256-byte aligned; work
 * enqueued on `stream`, nothing allocated or synchronised. Errors as for the boundary ops. */

/* Muon's Newton-Schulz coefficients: the quintic iteration X <- a X + b (X X^T) X + c (X X^T)^2 X
 * published with Muon (the paper cites Muon without restating them). */
#define RESBM_NS_A 3.4445f
#define RESBM_NS_B (-4.7750f)
#define RESBM_NS_C 2.0315f
#define RESBM_NS_EPS 1e-7f

/* Scratch bytes of `op` (RESBM_OP_EFFECTIVE_RANK or RESBM_OP_NEWTON_SCHULZ) for a rows x cols
 * matrix. INVALID_ARG for another op or a shape the kernels do not take. */
RESBM_API resbm_status resbm_matrix_workspace_bytes(int op, int64_t rows, int64_t cols, size_t *bytes);

/* Muon's orthogonalisation of a gradient (momentum) matrix G, rows x cols row-major, g_dtype
 * RESBM_F32 or RESBM_BF16: X_0 = G / (||G||_F + RESBM_NS_EPS), then `steps` (0..100; Muon uses 5)
 * Newton-Schulz steps X <- a X + (b A + c A A) X with A = X X^T, taken on the wide orientation
 * (for rows > cols the same iteration on X^T, i.e. X <- a X + X (b A + c A A) with A = X^T X).
 * X (rows x cols, bf16) receives the result; its singular vectors are G's and its singular values
 * are driven toward 1 (to about [0.7, 1.2]). The products run on the tensor cores with bf16
 * operands and fp32 accumulation, every iterate and product rounded to bf16, as Muon does. */
RESBM_API resbm_status resbm_newton_schulz(int64_t rows, int64_t cols, const void *G, int32_t g_dtype,
                                 int32_t steps, void *X, void *ws, size_t ws_bytes, void *stream);

/* The effective rank of a bf16 matrix W (rows x cols, row-major) as the appendix's spectral
 * analysis defines it, r_eff = sum_i sigma_i^2 / max_i sigma_i^2, computed as trace(S) /
 * lambda_max(S) for the Gram matrix S of W's smaller side (W^T W or W W^T; fp32 sums of the exact
 * bf16 products), lambda_max by power iteration on one CTA until the residual ||S v - lambda v||
 * is at most 1e-5 lambda ||v|| (at most 20000 iterations): some eigenvalue of S then lies within
 * 1e-5 (relative) of lambda (Bauer-Fike; the fp32 products put the residual's floor near 1e-6). `out` (device, 4 doubles): sigma_max^2, ||W||_F^2, r_eff, the iterations
 * taken. min(rows, cols) <= 4096. */
RESBM_API resbm_status resbm_effective_rank(int64_t rows, int64_t cols, const void *W, double *out,
                                  void *ws, size_t ws_bytes, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* RESBM_H */
