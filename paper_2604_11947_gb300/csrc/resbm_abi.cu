// resbm_abi.cu -- the C ABI of include/resbm.h: argument validation, scratch sizing and the
// choice between the tensor-core kernels and the portable CUDA-core kernels.
#include <cuda_runtime.h>
#include <stdint.h>
#include <math.h>
#include <string.h>

#include <atomic>
#include <map>
#include <memory>
#include <mutex>
#include <utility>

#include "internal.h"
#include "resbm.h"
#include "tc.h"

using namespace resbm;

namespace resbm {
static std::atomic<uint64_t> g_launches{0};
void count_launches(uint64_t n) { g_launches.fetch_add(n, std::memory_order_relaxed); }
}  // namespace resbm

namespace {

thread_local int g_last_cuda_error = 0;

resbm_status cuda_fail(cudaError_t e)
{
    g_last_cuda_error = (int)e;
    return RESBM_ERR_CUDA;
}

// The first columns of a row-major matrix between host and device when the host side is pinned
// and mapped: rows x w16 16-byte units, both sides rows pitch16 units apart, one unit per thread
// and grid step. Reading or writing the host rows in place over the host link beats a strided
// cudaMemcpy2DAsync of narrow rows (64-byte rows: 19 GB/s measured on GB300).
__global__ void k_copy_cols(const uint4 *__restrict__ src, uint4 *__restrict__ dst, int64_t rows, int64_t pitch16,
                            int64_t w16)
{
    const int64_t n = rows * w16;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t t = i / w16, j = i - t * w16;
        dst[t * pitch16 + j] = src[t * pitch16 + j];
    }
}

// The device address of a host buffer the device may access directly (page-locked and mapped:
// cudaHostAlloc, or cudaHostRegister with mapping), else null (pageable memory and errors).
void *mapped_host(const void *p)
{
    cudaPointerAttributes at{};
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
        cudaGetLastError();
        return nullptr;
    }
    return at.type == cudaMemoryTypeHost ? at.devicePointer : nullptr;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Side streams and events of resbm_boundary_step_host, created on first use for each (device,
// caller stream) and kept for the life of the process: creating and destroying streams in every
// call costs host time in the driver. An event re-recorded by the next call on the same caller
// stream is safe: a wait takes the state the event had when the wait was enqueued, and `mu`
// keeps two host threads from interleaving their enqueues on one entry.
struct SideStreams {
    cudaStream_t in = nullptr, out = nullptr;
    cudaEvent_t ev[5] = {};
    std::mutex mu;
};
cudaError_t side_streams(cudaStream_t caller, SideStreams **out)
{
    static std::mutex mu;
    static std::map<std::pair<int, cudaStream_t>, std::unique_ptr<SideStreams>> table;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> hold(mu);
    std::unique_ptr<SideStreams> &slot = table[{dev, caller}];
    if (!slot) {
        std::unique_ptr<SideStreams> s(new SideStreams);
        e = cudaStreamCreateWithFlags(&s->in, cudaStreamNonBlocking);
        if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&s->out, cudaStreamNonBlocking);
        for (int i = 0; i < 5 && e == cudaSuccess; ++i) e = cudaEventCreateWithFlags(&s->ev[i], cudaEventDisableTiming);
        if (e != cudaSuccess) {
            if (s->in) cudaStreamDestroy(s->in);
            if (s->out) cudaStreamDestroy(s->out);
            for (cudaEvent_t x : s->ev)
                if (x) cudaEventDestroy(x);
            table.erase({dev, caller});
            return e;
        }
        slot = std::move(s);
    }
    *out = slot.get();
    return cudaSuccess;
}

constexpr int kMaxDevices = 64;
std::atomic<int> g_sm_count[kMaxDevices];

resbm_status make_ctx(void *stream, Ctx *c)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e);
    int sms = (dev >= 0 && dev < kMaxDevices) ? g_sm_count[dev].load(std::memory_order_relaxed) : 0;
    if (sms <= 0) {
        e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (e != cudaSuccess) return cuda_fail(e);
        if (dev >= 0 && dev < kMaxDevices) g_sm_count[dev].store(sms, std::memory_order_relaxed);
    }
    c->stream = static_cast<cudaStream_t>(stream);
    c->device = dev;
    c->sm_count = sms;
    return RESBM_OK;
}

// SM count that sizes the scratch memory: the current device's, or kDefaultSms when no device
// can be queried (the tensor-core backward kernels keep one partial slot per CTA).
constexpr int kDefaultSms = 160;
int sizing_sms()
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        return kDefaultSms;
    }
    int sms = (dev >= 0 && dev < kMaxDevices) ? g_sm_count[dev].load(std::memory_order_relaxed) : 0;
    if (sms > 0) return sms;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0) {
        cudaGetLastError();
        return kDefaultSms;
    }
    if (dev >= 0 && dev < kMaxDevices) g_sm_count[dev].store(sms, std::memory_order_relaxed);
    return sms;
}

size_t elem_size(const resbm_desc &d) { return d.dtype == RESBM_BF16 ? 2 : 4; }

bool mul_ok(int64_t a, int64_t b) { return a >= 0 && b >= 0 && (a == 0 || b <= INT64_MAX / a); }

resbm_status check_desc(const resbm_desc *d)
{
    if (!d) return RESBM_ERR_INVALID_ARG;
    if (d->T < 0 || d->d < 1 || d->r < 1 || d->m < 1 || d->r > d->d) return RESBM_ERR_INVALID_ARG;
    if (d->dtype != RESBM_F32 && d->dtype != RESBM_BF16) return RESBM_ERR_INVALID_ARG;
    if (d->act != RESBM_ACT_SILU && d->act != RESBM_ACT_GELU_TANH && d->act != RESBM_ACT_IDENTITY)
        return RESBM_ERR_INVALID_ARG;
    if (d->merge_identity != 0 && d->merge_identity != 1) return RESBM_ERR_INVALID_ARG;
    if (d->flags & ~(RESBM_FLAG_GENERIC | RESBM_FLAG_LINEAR | RESBM_FLAG_GEMM)) return RESBM_ERR_INVALID_ARG;
    if ((d->flags & RESBM_FLAG_LINEAR) && d->m != d->r) return RESBM_ERR_INVALID_ARG;
    // every element count (and the byte counts derived from it) must fit in int64
    const int64_t big = INT64_MAX / 64;
    if (!mul_ok(d->T, d->d) || d->T * d->d > big || !mul_ok(d->T, d->m) || d->T * d->m > big ||
        !mul_ok(d->d, d->m) || d->d * d->m > big || !mul_ok(d->m, d->r) || d->m * d->r > big)
        return RESBM_ERR_INVALID_ARG;
    return RESBM_OK;
}

// A tensor argument: required non-null when it has elements, aligned to its element size.
bool ptr_ok(const void *p, size_t align, bool required)
{
    if (!p) return !required;
    return (reinterpret_cast<uintptr_t>(p) % align) == 0;
}

struct Range {
    uintptr_t lo, hi;
};
Range rng(const void *p, int64_t n, size_t es)
{
    uintptr_t a = reinterpret_cast<uintptr_t>(p);
    return Range{a, a + (uintptr_t)n * es};
}
bool overlaps(Range a, Range b)
{
    if (!a.lo || !b.lo || a.lo == a.hi || b.lo == b.hi) return false;
    return a.lo < b.hi && b.lo < a.hi;
}
template <size_t N> bool any_overlap(const Range (&outs)[N], const Range *ins, size_t nin)
{
    for (size_t i = 0; i < N; ++i) {
        for (size_t j = 0; j < nin; ++j)
            if (overlaps(outs[i], ins[j])) return true;
        for (size_t j = i + 1; j < N; ++j)
            if (overlaps(outs[i], outs[j])) return true;
    }
    return false;
}

// Which kernels run an op: the fused tensor-core kernels where they take the shape (unless a
// flag says otherwise), else the tensor-core GEMM chain, else the portable CUDA-core kernels.
bool use_tc(const resbm_desc &d, int op)
{
    return !(d.flags & (RESBM_FLAG_GENERIC | RESBM_FLAG_GEMM)) && tc_supported(d, op);
}
bool use_gemm(const resbm_desc &d, int op) { return !(d.flags & RESBM_FLAG_GENERIC) && gemm_supported(d, op); }

// ---- RESBM_FLAG_LINEAR ---------------------------------------------------------------------
// One linear layer per side runs as the two-layer path with identity second layers
// (We2 = Wd1 = I_r, phi = identity): exact, since multiplying by I_r and applying the identity
// function change no value. The identity matrix and two r x r gradient outputs nobody reads
// sit at the front of the workspace.
bool is_linear(const resbm_desc &d) { return (d.flags & RESBM_FLAG_LINEAR) != 0; }

resbm_desc two_layer(const resbm_desc &d)
{
    resbm_desc e = d;
    if (is_linear(d)) {
        e.act = RESBM_ACT_IDENTITY;
        e.flags &= ~RESBM_FLAG_LINEAR;
    }
    return e;
}

struct LinearWs {
    void *I;
    float *dW2, *dW1;
    void *inner;
    size_t bytes;
};
LinearWs carve_linear(const resbm_desc &d, void *ws)
{
    WsCarver w(ws);
    LinearWs l;
    l.I = w.take<char>((size_t)(d.r * d.r) * elem_size(d));
    l.dW2 = w.take<float>(d.r * d.r);
    l.dW1 = w.take<float>(d.r * d.r);
    l.inner = w.take<char>(0);
    l.bytes = w.used;
    return l;
}

size_t ws_for(const resbm_desc &d0, int op)
{
    if (op == RESBM_OP_RMSNORM_BWD) return rmsnorm_bwd_supported(d0) ? rmsnorm_bwd_ws_bytes(d0) : 0;
    if (op == RESBM_OP_DECODE_FWD_RMSNORM) {
        // the decoder forward's own scratch, or the fused form's row sums of squares
        const resbm_desc d = two_layer(d0);
        size_t b = ws_for(d0, RESBM_OP_DECODE_FWD);
        if (tc_supported(d, RESBM_OP_DECODE_FWD)) {
            const size_t f = (is_linear(d0) ? carve_linear(d0, nullptr).bytes : 0) + tc_rmsnorm_ws_bytes(d);
            if (f > b) b = f;
        }
        return b;
    }
    const resbm_desc d = two_layer(d0);
    size_t g = generic_ws_bytes(d, op);
    size_t t = tc_supported(d, op) ? tc_ws_bytes(d, op, sizing_sms()) : 0;
    size_t k = gemm_supported(d, op) ? gemm_ws_bytes(d, op, sizing_sms()) : 0;
    size_t inner = g > t ? g : t;
    if (k > inner) inner = k;
    return is_linear(d0) ? carve_linear(d0, nullptr).bytes + inner : inner;
}

size_t step_ws_bytes(const resbm_desc &d)
{
    WsCarver w(nullptr);
    w.take<float>(d.T * d.m);  // P when the caller passes none
    size_t inner = 0;
    for (int op = RESBM_OP_ENCODE_FWD; op <= RESBM_OP_ENCODE_BWD; ++op) {
        size_t b = ws_for(d, op);
        if (b > inner) inner = b;
    }
    w.take<char>(inner);
    return w.used;
}

size_t host_stage_bytes(const resbm_desc &d);   // resbm_boundary_step_host's workspace

resbm_status check_ws(const resbm_desc &d, int op, void *ws, size_t ws_bytes)
{
    size_t need = op == RESBM_OP_BOUNDARY_STEP_HOST ? host_stage_bytes(d)
                  : op == RESBM_OP_BOUNDARY_STEP    ? step_ws_bytes(d)
                                                    : ws_for(d, op);
    if (need == 0) return RESBM_OK;
    if (!ws || ws_bytes < need) return RESBM_ERR_WORKSPACE;
    if (reinterpret_cast<uintptr_t>(ws) % 256) return RESBM_ERR_INVALID_ARG;
    return RESBM_OK;
}

resbm_status zero_f32(float *p, int64_t n, cudaStream_t s)
{
    if (!p || n <= 0) return RESBM_OK;
    cudaError_t e = cudaMemsetAsync(p, 0, (size_t)n * sizeof(float), s);
    return e == cudaSuccess ? RESBM_OK : cuda_fail(e);
}

resbm_status finish(cudaError_t e) { return e == cudaSuccess ? RESBM_OK : cuda_fail(e); }

// ---- per-op validation (no GPU work) ---------------------------------------------------------
resbm_status validate_encode_fwd(const resbm_desc &d, const void *X, const void *F,
                                 const void *We1, const void *We2, const void *B,
                                 const float *P)
{
    const size_t es = elem_size(d);
    const bool t = d.T > 0;
    if (!ptr_ok(X, es, t) || !ptr_ok(F, es, t) || !ptr_ok(We1, es, true) ||
        !ptr_ok(We2, es, !is_linear(d)) || !ptr_ok(B, es, t) || !ptr_ok(P, 4, false))
        return RESBM_ERR_INVALID_ARG;
    const Range outs[] = {rng(B, d.T * d.r, es), rng(P, d.T * d.m, 4)};
    const Range ins[] = {rng(X, d.T * d.d, es), rng(F, d.T * d.d, es), rng(We1, d.d * d.m, es),
                         rng(We2, d.m * d.r, es)};
    return any_overlap(outs, ins, 4) ? RESBM_ERR_INVALID_ARG : RESBM_OK;
}

resbm_status validate_decode_fwd(const resbm_desc &d, const void *B, const void *Wd1,
                                 const void *Wd2, const void *Y)
{
    const size_t es = elem_size(d);
    const bool t = d.T > 0;
    if (!ptr_ok(B, es, t) || !ptr_ok(Wd1, es, !is_linear(d)) || !ptr_ok(Wd2, es, true) ||
        !ptr_ok(Y, es, t))
        return RESBM_ERR_INVALID_ARG;
    const Range outs[] = {rng(Y, d.T * d.d, es)};
    const Range ins[] = {rng(B, d.T * d.r, es), rng(Wd1, d.r * d.m, es), rng(Wd2, d.m * d.d, es)};
    return any_overlap(outs, ins, 3) ? RESBM_ERR_INVALID_ARG : RESBM_OK;
}

resbm_status validate_decode_fwd_rmsnorm(const resbm_desc &d, const void *B, const void *Wd1, const void *Wd2,
                                         const void *gamma, float eps, const void *Y, const void *N)
{
    const size_t es = elem_size(d);
    const bool t = d.T > 0;
    if (!ptr_ok(B, es, t) || !ptr_ok(Wd1, es, !is_linear(d)) || !ptr_ok(Wd2, es, true) || !ptr_ok(Y, es, t) ||
        !ptr_ok(N, es, t) || !ptr_ok(gamma, es, true) || !(eps >= 0.0f) || !(eps < INFINITY))
        return RESBM_ERR_INVALID_ARG;
    const Range outs[] = {rng(Y, d.T * d.d, es), rng(N, d.T * d.d, es)};
    const Range ins[] = {rng(B, d.T * d.r, es), rng(Wd1, d.r * d.m, es), rng(Wd2, d.m * d.d, es),
                         rng(gamma, d.d, es)};
    return any_overlap(outs, ins, 4) ? RESBM_ERR_INVALID_ARG : RESBM_OK;
}

resbm_status validate_decode_bwd(const resbm_desc &d, const void *dY, const void *B,
                                 const void *Wd1, const void *Wd2, const void *dB,
                                 const float *dWd1, const float *dWd2)
{
    const size_t es = elem_size(d);
    const bool t = d.T > 0;
    if (!ptr_ok(dY, es, t) || !ptr_ok(B, es, t) || !ptr_ok(Wd1, es, !is_linear(d)) ||
        !ptr_ok(Wd2, es, true) || !ptr_ok(dB, es, t) || !ptr_ok(dWd1, 4, !is_linear(d)) ||
        !ptr_ok(dWd2, 4, true))
        return RESBM_ERR_INVALID_ARG;
    const Range outs[] = {rng(dB, d.T * d.r, es), rng(dWd1, d.r * d.m, 4), rng(dWd2, d.m * d.d, 4)};
    const Range ins[] = {rng(dY, d.T * d.d, es), rng(B, d.T * d.r, es), rng(Wd1, d.r * d.m, es),
                         rng(Wd2, d.m * d.d, es)};
    return any_overlap(outs, ins, 4) ? RESBM_ERR_INVALID_ARG : RESBM_OK;
}

resbm_status validate_encode_bwd(const resbm_desc &d, const void *dB, const void *F,
                                 const float *P, const void *We1, const void *We2,
                                 const void *dF, const void *dX, const float *dWe1,
                                 const float *dWe2)
{
    const size_t es = elem_size(d);
    const bool t = d.T > 0;
    if (!ptr_ok(dB, es, t) || !ptr_ok(F, es, t) || !ptr_ok(P, 4, false) ||
        !ptr_ok(We1, es, true) || !ptr_ok(We2, es, !is_linear(d)) || !ptr_ok(dF, es, t) ||
        !ptr_ok(dX, es, false) || !ptr_ok(dWe1, 4, true) || !ptr_ok(dWe2, 4, !is_linear(d)))
        return RESBM_ERR_INVALID_ARG;
    const Range outs[] = {rng(dF, d.T * d.d, es), rng(dX, d.T * d.d, es), rng(dWe1, d.d * d.m, 4),
                          rng(dWe2, d.m * d.r, 4)};
    const Range ins[] = {rng(dB, d.T * d.r, es), rng(F, d.T * d.d, es), rng(P, d.T * d.m, 4),
                         rng(We1, d.d * d.m, es), rng(We2, d.m * d.r, es)};
    return any_overlap(outs, ins, 5) ? RESBM_ERR_INVALID_ARG : RESBM_OK;
}

// ---- per-op execution (after validation) -----------------------------------------------------
// A tensor-core launcher answers cudaErrorNotSupported (before launching anything) when it
// cannot take the call, e.g. for pointers that are not 16-byte aligned; the portable kernels run.
resbm_status run_encode_fwd(const resbm_desc &d, const void *X, const void *F, const void *We1,
                            const void *We2, void *B, float *P, void *ws, const Ctx &c)
{
    if (d.T == 0) return RESBM_OK;
    if (use_tc(d, RESBM_OP_ENCODE_FWD)) {
        cudaError_t e = tc_encode_fwd(d, X, F, We1, We2, B, P, ws, c);
        if (e != cudaErrorNotSupported) return finish(e);
    }
    if (use_gemm(d, RESBM_OP_ENCODE_FWD)) {
        cudaError_t e = gemm_encode_fwd(d, X, F, We1, We2, B, P, ws, c);
        if (e != cudaErrorNotSupported) return finish(e);
    }
    return finish(generic_encode_fwd(d, X, F, We1, We2, B, P, ws, c));
}

// on_tc (nullable): set when the tensor-core kernel (one launch, no scratch) ran
resbm_status run_decode_fwd(const resbm_desc &d, const void *B, const void *Wd1, const void *Wd2,
                            void *Y, void *ws, const Ctx &c, bool *on_tc = nullptr)
{
    if (on_tc) *on_tc = false;
    if (d.T == 0) return RESBM_OK;
    if (use_tc(d, RESBM_OP_DECODE_FWD)) {
        cudaError_t e = tc_decode_fwd(d, B, Wd1, Wd2, Y, ws, c);
        if (e != cudaErrorNotSupported) {
            if (on_tc) *on_tc = e == cudaSuccess;
            return finish(e);
        }
    }
    if (use_gemm(d, RESBM_OP_DECODE_FWD)) {
        cudaError_t e = gemm_decode_fwd(d, B, Wd1, Wd2, Y, ws, c);
        if (e != cudaErrorNotSupported) return finish(e);
    }
    return finish(generic_decode_fwd(d, B, Wd1, Wd2, Y, ws, c));
}

// after_independent: see tc_decode_bwd (the boundary step, right after its decoder forward)
resbm_status run_decode_bwd(const resbm_desc &d, const void *dY, const void *B, const void *Wd1,
                            const void *Wd2, void *dB, float *dWd1, float *dWd2, void *ws,
                            const Ctx &c, bool after_independent = false)
{
    if (d.T == 0) {
        resbm_status s = zero_f32(dWd1, d.r * d.m, c.stream);
        return s != RESBM_OK ? s : zero_f32(dWd2, d.m * d.d, c.stream);
    }
    if (use_tc(d, RESBM_OP_DECODE_BWD)) {
        cudaError_t e = tc_decode_bwd(d, dY, B, Wd1, Wd2, dB, dWd1, dWd2, ws, c, after_independent);
        if (e != cudaErrorNotSupported) return finish(e);
    }
    if (use_gemm(d, RESBM_OP_DECODE_BWD)) {
        cudaError_t e = gemm_decode_bwd(d, dY, B, Wd1, Wd2, dB, dWd1, dWd2, ws, c);
        if (e != cudaErrorNotSupported) return finish(e);
    }
    return finish(generic_decode_bwd(d, dY, B, Wd1, Wd2, dB, dWd1, dWd2, ws, c));
}

resbm_status run_encode_bwd(const resbm_desc &d, const void *dB, const void *F, const float *P,
                            const void *We1, const void *We2, void *dF, void *dX, float *dWe1,
                            float *dWe2, void *ws, const Ctx &c)
{
    if (d.T == 0) {
        resbm_status s = zero_f32(dWe1, d.d * d.m, c.stream);
        return s != RESBM_OK ? s : zero_f32(dWe2, d.m * d.r, c.stream);
    }
    if (use_tc(d, RESBM_OP_ENCODE_BWD)) {
        cudaError_t e = tc_encode_bwd(d, dB, F, P, We1, We2, dF, dX, dWe1, dWe2, ws, c);
        if (e != cudaErrorNotSupported) return finish(e);
    }
    if (use_gemm(d, RESBM_OP_ENCODE_BWD)) {
        cudaError_t e = gemm_encode_bwd(d, dB, F, P, We1, We2, dF, dX, dWe1, dWe2, ws, c);
        if (e != cudaErrorNotSupported) return finish(e);
    }
    return finish(generic_encode_bwd(d, dB, F, P, We1, We2, dF, dX, dWe1, dWe2, ws, c));
}

// ---- the four ops on either form (after validation) -----------------------------------------
resbm_status exec_encode_fwd(const resbm_desc &d, const void *X, const void *F, const void *We1,
                             const void *We2, void *B, float *P, void *ws, const Ctx &c)
{
    if (!is_linear(d)) return run_encode_fwd(d, X, F, We1, We2, B, P, ws, c);
    const LinearWs l = carve_linear(d, ws);
    resbm_status s = finish(fill_identity(d, l.I, c));
    return s != RESBM_OK ? s : run_encode_fwd(two_layer(d), X, F, We1, l.I, B, P, l.inner, c);
}

resbm_status exec_decode_fwd(const resbm_desc &d, const void *B, const void *Wd1, const void *Wd2,
                             void *Y, void *ws, const Ctx &c)
{
    if (!is_linear(d)) return run_decode_fwd(d, B, Wd1, Wd2, Y, ws, c);
    const LinearWs l = carve_linear(d, ws);
    resbm_status s = finish(fill_identity(d, l.I, c));
    return s != RESBM_OK ? s : run_decode_fwd(two_layer(d), B, l.I, Wd2, Y, l.inner, c);
}

// the fused tensor-core form where the decoder forward runs on the fused kernels, else the
// decoder forward followed by the norm over the stored Y
resbm_status run_decode_fwd_rmsnorm(const resbm_desc &d, const void *B, const void *Wd1, const void *Wd2,
                                    const void *gamma, float eps, void *Y, void *N, void *ws, const Ctx &c)
{
    if (d.T == 0) return RESBM_OK;
    if (use_tc(d, RESBM_OP_DECODE_FWD)) {
        cudaError_t e = tc_decode_fwd_rmsnorm(d, B, Wd1, Wd2, gamma, eps, Y, N, ws, c);
        if (e != cudaErrorNotSupported) return finish(e);
    }
    resbm_status s = run_decode_fwd(d, B, Wd1, Wd2, Y, ws, c);
    return s != RESBM_OK ? s : finish(generic_rmsnorm(d, Y, gamma, eps, N, c));
}

resbm_status exec_decode_fwd_rmsnorm(const resbm_desc &d, const void *B, const void *Wd1, const void *Wd2,
                                     const void *gamma, float eps, void *Y, void *N, void *ws, const Ctx &c)
{
    if (!is_linear(d)) return run_decode_fwd_rmsnorm(d, B, Wd1, Wd2, gamma, eps, Y, N, ws, c);
    const LinearWs l = carve_linear(d, ws);
    resbm_status s = finish(fill_identity(d, l.I, c));
    return s != RESBM_OK ? s : run_decode_fwd_rmsnorm(two_layer(d), B, l.I, Wd2, gamma, eps, Y, N, l.inner, c);
}

resbm_status exec_decode_bwd(const resbm_desc &d, const void *dY, const void *B, const void *Wd1,
                             const void *Wd2, void *dB, float *dWd1, float *dWd2, void *ws,
                             const Ctx &c)
{
    if (!is_linear(d)) return run_decode_bwd(d, dY, B, Wd1, Wd2, dB, dWd1, dWd2, ws, c);
    const LinearWs l = carve_linear(d, ws);
    resbm_status s = finish(fill_identity(d, l.I, c));
    return s != RESBM_OK ? s
                         : run_decode_bwd(two_layer(d), dY, B, l.I, Wd2, dB, l.dW1, dWd2, l.inner, c);
}

resbm_status exec_encode_bwd(const resbm_desc &d, const void *dB, const void *F, const float *P,
                             const void *We1, const void *We2, void *dF, void *dX, float *dWe1,
                             float *dWe2, void *ws, const Ctx &c)
{
    if (!is_linear(d)) return run_encode_bwd(d, dB, F, P, We1, We2, dF, dX, dWe1, dWe2, ws, c);
    const LinearWs l = carve_linear(d, ws);
    resbm_status s = finish(fill_identity(d, l.I, c));
    return s != RESBM_OK ? s
                         : run_encode_bwd(two_layer(d), dB, F, P, We1, l.I, dF, dX, dWe1, l.dW2,
                                          l.inner, c);
}

// ---- the boundary step (device or host buffers) ---------------------------------------------
// All four stages' checks, and no output overlapping another output or an input.
resbm_status validate_step(const resbm_desc &d, const resbm_step_args *a)
{
    resbm_status s = validate_encode_fwd(d, a->X, a->F, a->We1, a->We2, a->B, a->P);
    if (s == RESBM_OK) s = validate_decode_fwd(d, a->B, a->Wd1, a->Wd2, a->Y);
    if (s == RESBM_OK) s = validate_decode_bwd(d, a->dY, a->B, a->Wd1, a->Wd2, a->dB, a->dWd1, a->dWd2);
    if (s == RESBM_OK)
        s = validate_encode_bwd(d, a->dB, a->F, a->P, a->We1, a->We2, a->dF, a->dX, a->dWe1, a->dWe2);
    if (s == RESBM_OK) {
        const size_t es = elem_size(d);
        const Range outs[] = {rng(a->B, d.T * d.r, es), rng(a->P, d.T * d.m, 4),
                              rng(a->Y, d.T * d.d, es), rng(a->dB, d.T * d.r, es),
                              rng(a->dF, d.T * d.d, es), rng(a->dX, d.T * d.d, es),
                              rng(a->dWe1, d.d * d.m, 4), rng(a->dWe2, d.m * d.r, 4),
                              rng(a->dWd1, d.r * d.m, 4), rng(a->dWd2, d.m * d.d, 4)};
        const Range ins[] = {rng(a->X, d.T * d.d, es), rng(a->F, d.T * d.d, es),
                             rng(a->dY, d.T * d.d, es)};
        if (any_overlap(outs, ins, 3)) s = RESBM_ERR_INVALID_ARG;
    }
    return s;
}

// Enqueues the four stages on c.stream (device pointers, validated). With fwd_done, records it
// after the forward stages; with bwd_ready, the backward stages wait for it.
resbm_status enqueue_step(const resbm_desc &d, const resbm_step_args &a, void *ws, const Ctx &c,
                          cudaEvent_t fwd_done, cudaEvent_t bwd_ready)
{
    WsCarver w(ws);
    float *P = a.P ? a.P : w.take<float>(d.T * d.m);
    void *inner = w.take<char>(0);
    const void *We2 = a.We2, *Wd1 = a.Wd1;
    float *dWe2 = a.dWe2, *dWd1 = a.dWd1;
    const resbm_desc e = two_layer(d);
    resbm_status s = RESBM_OK;
    if (is_linear(d)) {
        const LinearWs l = carve_linear(d, inner);
        s = finish(fill_identity(d, l.I, c));
        We2 = Wd1 = l.I;
        dWe2 = l.dW2;
        dWd1 = l.dW1;
        inner = l.inner;
    }
    if (s == RESBM_OK) s = run_encode_fwd(e, a.X, a.F, a.We1, We2, a.B, P, inner, c);
    bool dec_fwd_tc = false;
    if (s == RESBM_OK) s = run_decode_fwd(e, a.B, Wd1, a.Wd2, a.Y, inner, c, &dec_fwd_tc);
    if (s == RESBM_OK && fwd_done) s = finish(cudaEventRecord(fwd_done, c.stream));
    if (s == RESBM_OK && bwd_ready) s = finish(cudaStreamWaitEvent(c.stream, bwd_ready, 0));
    // the decoder backward reads dY and B, not the decoder forward's Y, and the tensor-core
    // decoder forward uses no scratch: with nothing queued between the two kernels the backward
    // starts as the forward's CTAs leave (tc_decode_bwd)
    const bool overlap = dec_fwd_tc && fwd_done == nullptr && bwd_ready == nullptr;
    if (s == RESBM_OK) s = run_decode_bwd(e, a.dY, a.B, Wd1, a.Wd2, a.dB, dWd1, a.dWd2, inner, c, overlap);
    if (s == RESBM_OK)
        s = run_encode_bwd(e, a.dB, a.F, P, a.We1, We2, a.dF, a.dX, a.dWe1, dWe2, inner, c);
    return s;
}

// Device staging of resbm_boundary_step_host: a device copy of every tensor of the step (X and
// dX full T x d, of which only the first r columns are copied), then the step's own scratch.
struct HostStage {
    resbm_step_args dev;
    void *inner;
    size_t bytes;
};
HostStage carve_host_stage(const resbm_desc &d, void *ws, const resbm_step_args &host)
{
    const size_t es = elem_size(d);
    const int64_t T = d.T, D = d.d, r = d.r, m = d.m;
    WsCarver w(ws);
    HostStage h{};
    h.dev.X = w.take<char>((size_t)(T * D) * es);
    h.dev.F = w.take<char>((size_t)(T * D) * es);
    h.dev.dY = w.take<char>((size_t)(T * D) * es);
    h.dev.We1 = w.take<char>((size_t)(D * m) * es);
    h.dev.We2 = w.take<char>((size_t)(m * r) * es);
    h.dev.Wd1 = w.take<char>((size_t)(r * m) * es);
    h.dev.Wd2 = w.take<char>((size_t)(m * D) * es);
    h.dev.B = w.take<char>((size_t)(T * r) * es);
    h.dev.P = w.take<float>(T * m);
    h.dev.Y = w.take<char>((size_t)(T * D) * es);
    h.dev.dB = w.take<char>((size_t)(T * r) * es);
    h.dev.dF = w.take<char>((size_t)(T * D) * es);
    void *dX = w.take<char>((size_t)(T * D) * es);
    h.dev.dX = host.dX ? dX : nullptr;
    h.dev.dWe1 = w.take<float>(D * m);
    h.dev.dWe2 = w.take<float>(m * r);
    h.dev.dWd1 = w.take<float>(r * m);
    h.dev.dWd2 = w.take<float>(m * D);
    if (is_linear(d)) {   // one linear layer: the second-layer weights are not read
        h.dev.We2 = h.dev.Wd1 = nullptr;
        h.dev.dWe2 = h.dev.dWd1 = nullptr;
    }
    h.inner = w.take<char>(0);
    w.take<char>(step_ws_bytes(d));
    h.bytes = w.used;
    return h;
}

size_t host_stage_bytes(const resbm_desc &d) { return carve_host_stage(d, nullptr, resbm_step_args{}).bytes; }

// ---- fixed scratch of resbm_decode_bwd_noalloc -----------------------------------------------
// One array per device, reserved with the library's device code; its address is looked up on
// the first call on each device and kept (all host threads share the cached value).
static __device__ __align__(256) unsigned char g_static_scratch[RESBM_STATIC_SCRATCH_BYTES];
std::atomic<void *> g_static_scratch_ptr[kMaxDevices];

resbm_status static_scratch(int dev, void **out)
{
    if (dev < 0 || dev >= kMaxDevices) return RESBM_ERR_UNSUPPORTED;
    void *p = g_static_scratch_ptr[dev].load(std::memory_order_acquire);
    if (!p) {
        cudaError_t e = cudaGetSymbolAddress(&p, g_static_scratch);
        if (e != cudaSuccess) return cuda_fail(e);
        g_static_scratch_ptr[dev].store(p, std::memory_order_release);
    }
    *out = p;
    return RESBM_OK;
}

}  // namespace

extern "C" {

const char *resbm_version(void) { return "resbm 0.1.0 sm_103a"; }

const char *resbm_status_string(resbm_status s)
{
    switch (s) {
    case RESBM_OK: return "RESBM_OK";
    case RESBM_ERR_INVALID_ARG: return "RESBM_ERR_INVALID_ARG";
    case RESBM_ERR_UNSUPPORTED: return "RESBM_ERR_UNSUPPORTED";
    case RESBM_ERR_WORKSPACE: return "RESBM_ERR_WORKSPACE";
    case RESBM_ERR_CUDA: return "RESBM_ERR_CUDA";
    }
    return "RESBM_ERR_UNKNOWN";
}

int resbm_last_cuda_error(void) { return g_last_cuda_error; }

uint64_t resbm_kernel_launches(void) { return g_launches.load(std::memory_order_relaxed); }

resbm_status resbm_device_error(unsigned int *code, int clear)
{
    if (!code) return RESBM_ERR_INVALID_ARG;
    *code = 0;
    cudaError_t e = tc_device_error(code, clear != 0);
    return e == cudaSuccess ? RESBM_OK : cuda_fail(e);
}

resbm_status resbm_selftest_wait_timeout(void *stream)
{
    Ctx c;
    resbm_status s = make_ctx(stream, &c);
    return s != RESBM_OK ? s : finish(tc_wait_selftest(c));
}

resbm_status resbm_measure_hbm_form(int form, const void *a, void *b, int64_t bytes, void *stream)
{
    constexpr int64_t kMiB = int64_t(1) << 20;
    if (form < RESBM_HBM_READ_V4 || form > RESBM_HBM_WRITE_TMA_2D_TILES || bytes < kMiB || bytes % kMiB != 0 ||
        bytes / 8192 > INT32_MAX || !a || !b || !aligned16(a) || !aligned16(b) ||
        overlaps(rng(a, bytes, 1), rng(b, bytes, 1)))
        return RESBM_ERR_INVALID_ARG;
    Ctx c;
    resbm_status s = make_ctx(stream, &c);
    return s != RESBM_OK ? s : finish(tc_hbm_form(form, a, b, bytes, c));
}

resbm_status resbm_workspace_bytes(const resbm_desc *desc, int op, size_t *bytes)
{
    resbm_status s = check_desc(desc);
    if (s != RESBM_OK) return s;
    if (!bytes || op < RESBM_OP_ENCODE_FWD ||
        (op > RESBM_OP_BOUNDARY_STEP_HOST && op != RESBM_OP_DECODE_FWD_RMSNORM && op != RESBM_OP_RMSNORM_BWD))
        return RESBM_ERR_INVALID_ARG;
    *bytes = op == RESBM_OP_BOUNDARY_STEP_HOST ? host_stage_bytes(*desc)
             : op == RESBM_OP_BOUNDARY_STEP    ? step_ws_bytes(*desc)
                                               : ws_for(*desc, op);
    return RESBM_OK;
}

resbm_status resbm_encode_fwd(const resbm_desc *desc, const void *X, const void *F,
                              const void *We1, const void *We2, void *B, float *P_save,
                              void *ws, size_t ws_bytes, void *stream)
{
    resbm_status s = check_desc(desc);
    if (s == RESBM_OK) s = validate_encode_fwd(*desc, X, F, We1, We2, B, P_save);
    if (s == RESBM_OK) s = check_ws(*desc, RESBM_OP_ENCODE_FWD, ws, ws_bytes);
    Ctx c;
    if (s == RESBM_OK) s = make_ctx(stream, &c);
    if (s == RESBM_OK) s = exec_encode_fwd(*desc, X, F, We1, We2, B, P_save, ws, c);
    return s;
}

resbm_status resbm_decode_fwd(const resbm_desc *desc, const void *B, const void *Wd1,
                              const void *Wd2, void *Y, void *ws, size_t ws_bytes, void *stream)
{
    resbm_status s = check_desc(desc);
    if (s == RESBM_OK) s = validate_decode_fwd(*desc, B, Wd1, Wd2, Y);
    if (s == RESBM_OK) s = check_ws(*desc, RESBM_OP_DECODE_FWD, ws, ws_bytes);
    Ctx c;
    if (s == RESBM_OK) s = make_ctx(stream, &c);
    if (s == RESBM_OK) s = exec_decode_fwd(*desc, B, Wd1, Wd2, Y, ws, c);
    return s;
}

resbm_status resbm_decode_fwd_rmsnorm(const resbm_desc *desc, const void *B, const void *Wd1, const void *Wd2,
                                      const void *gamma, float eps, void *Y, void *N, void *ws, size_t ws_bytes,
                                      void *stream)
{
    resbm_status s = check_desc(desc);
    if (s == RESBM_OK) s = validate_decode_fwd_rmsnorm(*desc, B, Wd1, Wd2, gamma, eps, Y, N);
    if (s == RESBM_OK) s = check_ws(*desc, RESBM_OP_DECODE_FWD_RMSNORM, ws, ws_bytes);
    Ctx c;
    if (s == RESBM_OK) s = make_ctx(stream, &c);
    if (s == RESBM_OK) s = exec_decode_fwd_rmsnorm(*desc, B, Wd1, Wd2, gamma, eps, Y, N, ws, c);
    return s;
}

resbm_status resbm_rmsnorm_bwd(const resbm_desc *desc, const void *Y, const void *gamma, float eps, const void *dN,
                               const void *dY, void *dY_out, float *dgamma, void *ws, size_t ws_bytes, void *stream)
{
    resbm_status s = check_desc(desc);
    if (s != RESBM_OK) return s;
    const resbm_desc &d = *desc;
    if (!rmsnorm_bwd_supported(d)) return RESBM_ERR_UNSUPPORTED;
    const size_t es = elem_size(d);
    const bool t = d.T > 0;
    if (!ptr_ok(Y, es, t) || !ptr_ok(gamma, es, true) || !ptr_ok(dN, es, t) || !ptr_ok(dY, es, false) ||
        !ptr_ok(dY_out, es, t) || !ptr_ok(dgamma, 4, true) || !(eps >= 0.0f) || !(eps < INFINITY))
        return RESBM_ERR_INVALID_ARG;
    // dY_out may be dY itself (in place); otherwise no output overlaps an input or the other output
    const Range outs[] = {rng(dY_out, d.T * d.d, es), rng(dgamma, d.d, 4)};
    const Range ins[] = {rng(Y, d.T * d.d, es), rng(gamma, d.d, es), rng(dN, d.T * d.d, es),
                         rng(dY == dY_out ? nullptr : dY, d.T * d.d, es)};
    if (any_overlap(outs, ins, 4)) return RESBM_ERR_INVALID_ARG;
    if (dY && dY != dY_out && overlaps(rng(dY, d.T * d.d, es), rng(dY_out, d.T * d.d, es)))
        return RESBM_ERR_INVALID_ARG;
    s = check_ws(d, RESBM_OP_RMSNORM_BWD, ws, ws_bytes);
    Ctx c;
    if (s == RESBM_OK) s = make_ctx(stream, &c);
    if (s == RESBM_OK) s = finish(generic_rmsnorm_bwd(d, Y, gamma, eps, dN, dY, dY_out, dgamma, ws, c));
    return s;
}

resbm_status resbm_decode_bwd(const resbm_desc *desc, const void *dY, const void *B,
                              const void *Wd1, const void *Wd2, void *dB, float *dWd1,
                              float *dWd2, void *ws, size_t ws_bytes, void *stream)
{
    resbm_status s = check_desc(desc);
    if (s == RESBM_OK) s = validate_decode_bwd(*desc, dY, B, Wd1, Wd2, dB, dWd1, dWd2);
    if (s == RESBM_OK) s = check_ws(*desc, RESBM_OP_DECODE_BWD, ws, ws_bytes);
    Ctx c;
    if (s == RESBM_OK) s = make_ctx(stream, &c);
    if (s == RESBM_OK) s = exec_decode_bwd(*desc, dY, B, Wd1, Wd2, dB, dWd1, dWd2, ws, c);
    return s;
}

resbm_status resbm_decode_bwd_noalloc(const resbm_desc *desc, const void *dY, const void *B,
                                      const void *Wd1, const void *Wd2, void *dB, float *dWd1,
                                      float *dWd2, void *stream)
{
    resbm_status s = check_desc(desc);
    if (s == RESBM_OK) s = validate_decode_bwd(*desc, dY, B, Wd1, Wd2, dB, dWd1, dWd2);
    if (s == RESBM_OK && ws_for(*desc, RESBM_OP_DECODE_BWD) > RESBM_STATIC_SCRATCH_BYTES)
        s = RESBM_ERR_WORKSPACE;
    Ctx c;
    if (s == RESBM_OK) s = make_ctx(stream, &c);
    void *ws = nullptr;
    if (s == RESBM_OK) s = static_scratch(c.device, &ws);
    if (s == RESBM_OK) s = exec_decode_bwd(*desc, dY, B, Wd1, Wd2, dB, dWd1, dWd2, ws, c);
    return s;
}

resbm_status resbm_encode_bwd(const resbm_desc *desc, const void *dB, const void *F,
                              const float *P_save, const void *We1, const void *We2, void *dF,
                              void *dX, float *dWe1, float *dWe2, void *ws, size_t ws_bytes,
                              void *stream)
{
    resbm_status s = check_desc(desc);
    if (s == RESBM_OK)
        s = validate_encode_bwd(*desc, dB, F, P_save, We1, We2, dF, dX, dWe1, dWe2);
    if (s == RESBM_OK) s = check_ws(*desc, RESBM_OP_ENCODE_BWD, ws, ws_bytes);
    Ctx c;
    if (s == RESBM_OK) s = make_ctx(stream, &c);
    if (s == RESBM_OK)
        s = exec_encode_bwd(*desc, dB, F, P_save, We1, We2, dF, dX, dWe1, dWe2, ws, c);
    return s;
}

resbm_status resbm_boundary_step(const resbm_desc *desc, const resbm_step_args *a, void *ws,
                                 size_t ws_bytes, void *stream)
{
    resbm_status s = check_desc(desc);
    if (s != RESBM_OK) return s;
    if (!a) return RESBM_ERR_INVALID_ARG;
    const resbm_desc &d = *desc;
    s = check_ws(d, RESBM_OP_BOUNDARY_STEP, ws, ws_bytes);
    if (s == RESBM_OK) s = validate_step(d, a);
    Ctx c;
    if (s == RESBM_OK) s = make_ctx(stream, &c);
    return s == RESBM_OK ? enqueue_step(d, *a, ws, c, nullptr, nullptr) : s;
}

resbm_status resbm_ffn_down_encode_workspace_bytes(const resbm_desc *desc, int64_t f, size_t *bytes)
{
    resbm_status s = check_desc(desc);
    if (s != RESBM_OK) return s;
    if (!bytes || f < 1) return RESBM_ERR_INVALID_ARG;
    if (!ffn_encode_supported(*desc, f)) return RESBM_ERR_UNSUPPORTED;
    *bytes = ffn_encode_ws_bytes(*desc, f);
    return RESBM_OK;
}

resbm_status resbm_ffn_down_encode_fwd(const resbm_desc *desc, int64_t f, const void *H, const void *W2, const void *X,
                                       const void *We1, const void *We2, void *B, float *P_save, void *F_out,
                                       void *ws, size_t ws_bytes, void *stream)
{
    resbm_status s = check_desc(desc);
    if (s != RESBM_OK) return s;
    const resbm_desc &d = *desc;
    if (f < 1 || !mul_ok(d.T, f) || !mul_ok(f, d.d)) return RESBM_ERR_INVALID_ARG;
    if (!ffn_encode_supported(d, f)) return RESBM_ERR_UNSUPPORTED;
    const bool t = d.T > 0;
    if (!ptr_ok(H, 2, t) || !ptr_ok(W2, 2, true) || !ptr_ok(X, 2, t) || !ptr_ok(We1, 2, true) ||
        !ptr_ok(We2, 2, true) || !ptr_ok(B, 2, t) || !ptr_ok(P_save, 4, false) || !ptr_ok(F_out, 2, false))
        return RESBM_ERR_INVALID_ARG;
    const Range outs[] = {rng(B, d.T * d.r, 2), rng(P_save, d.T * d.m, 4), rng(F_out, d.T * d.d, 2)};
    const Range ins[] = {rng(H, d.T * f, 2), rng(W2, f * d.d, 2), rng(X, d.T * d.d, 2), rng(We1, d.d * d.m, 2),
                         rng(We2, d.m * d.r, 2)};
    if (any_overlap(outs, ins, 5)) return RESBM_ERR_INVALID_ARG;
    const size_t need = ffn_encode_ws_bytes(d, f);
    if (!ws || ws_bytes < need) return RESBM_ERR_WORKSPACE;
    if (reinterpret_cast<uintptr_t>(ws) % 256) return RESBM_ERR_INVALID_ARG;
    Ctx c;
    s = make_ctx(stream, &c);
    if (s != RESBM_OK || d.T == 0) return s;
    const cudaError_t e = tc_ffn_down_encode(d, f, H, W2, X, We1, We2, B, P_save, F_out, ws, c);
    return e == cudaErrorNotSupported ? RESBM_ERR_UNSUPPORTED : finish(e);
}

resbm_status resbm_matrix_workspace_bytes(int op, int64_t rows, int64_t cols, size_t *bytes)
{
    if (!bytes || (op != RESBM_OP_EFFECTIVE_RANK && op != RESBM_OP_NEWTON_SCHULZ)) return RESBM_ERR_INVALID_ARG;
    if (!matrix_supported(rows, cols)) return RESBM_ERR_INVALID_ARG;
    *bytes = matrix_ws_bytes(op, rows, cols, sizing_sms());
    return RESBM_OK;
}

resbm_status resbm_newton_schulz(int64_t rows, int64_t cols, const void *G, int32_t g_dtype, int32_t steps, void *X,
                                 void *ws, size_t ws_bytes, void *stream)
{
    if (!matrix_supported(rows, cols) || steps < 0 || steps > 100 || (g_dtype != RESBM_F32 && g_dtype != RESBM_BF16))
        return RESBM_ERR_INVALID_ARG;
    const size_t es = g_dtype == RESBM_F32 ? 4 : 2;
    if (!G || !X || !aligned16(G) || !aligned16(X)) return RESBM_ERR_INVALID_ARG;
    if (overlaps(rng(G, rows * cols, es), rng(X, rows * cols, 2))) return RESBM_ERR_INVALID_ARG;
    const size_t need = matrix_ws_bytes(RESBM_OP_NEWTON_SCHULZ, rows, cols, sizing_sms());
    if (!ws || ws_bytes < need) return RESBM_ERR_WORKSPACE;
    if (reinterpret_cast<uintptr_t>(ws) % 256) return RESBM_ERR_INVALID_ARG;
    Ctx c;
    resbm_status s = make_ctx(stream, &c);
    if (s != RESBM_OK) return s;
    const float coef[3] = {RESBM_NS_A, RESBM_NS_B, RESBM_NS_C};
    const cudaError_t e = tc_newton_schulz(rows, cols, G, g_dtype == RESBM_F32, steps, coef, RESBM_NS_EPS, X, ws, c);
    return e == cudaErrorNotSupported ? RESBM_ERR_UNSUPPORTED : finish(e);
}

resbm_status resbm_effective_rank(int64_t rows, int64_t cols, const void *W, double *out, void *ws, size_t ws_bytes,
                                  void *stream)
{
    if (!matrix_supported(rows, cols) || (rows < cols ? rows : cols) > 4096) return RESBM_ERR_INVALID_ARG;
    if (!W || !out || !aligned16(W) || (reinterpret_cast<uintptr_t>(out) % 8)) return RESBM_ERR_INVALID_ARG;
    const size_t need = matrix_ws_bytes(RESBM_OP_EFFECTIVE_RANK, rows, cols, sizing_sms());
    if (!ws || ws_bytes < need) return RESBM_ERR_WORKSPACE;
    if (reinterpret_cast<uintptr_t>(ws) % 256) return RESBM_ERR_INVALID_ARG;
    Ctx c;
    resbm_status s = make_ctx(stream, &c);
    if (s != RESBM_OK) return s;
    const cudaError_t e = tc_effective_rank(rows, cols, W, out, ws, c);
    return e == cudaErrorNotSupported ? RESBM_ERR_UNSUPPORTED : finish(e);
}

resbm_status resbm_boundary_step_host(const resbm_desc *desc, const resbm_step_args *a, void *ws,
                                      size_t ws_bytes, void *stream)
{
    resbm_status s = check_desc(desc);
    if (s != RESBM_OK) return s;
    if (!a) return RESBM_ERR_INVALID_ARG;
    const resbm_desc &d = *desc;
    s = check_ws(d, RESBM_OP_BOUNDARY_STEP_HOST, ws, ws_bytes);
    if (s == RESBM_OK) s = validate_step(d, a);
    Ctx c;
    if (s == RESBM_OK) s = make_ctx(stream, &c);
    if (s != RESBM_OK) return s;
    const HostStage hs = carve_host_stage(d, ws, *a);
    const resbm_step_args &dv = hs.dev;
    const size_t es = elem_size(d);
    const int64_t T = d.T, D = d.d, r = d.r, m = d.m;
    const bool lin = is_linear(d);
    // two side streams, forked from and joined back into the caller's stream; kept per
    // (device, caller stream) across calls, one call's enqueue at a time
    SideStreams *side = nullptr;
    cudaError_t e = side_streams(c.stream, &side);
    if (e != cudaSuccess) return cuda_fail(e);
    std::lock_guard<std::mutex> hold(side->mu);
    cudaStream_t s_in = side->in, s_out = side->out;
    cudaEvent_t fork = side->ev[0], dy_in = side->ev[1], fwd_done = side->ev[2], out_done = side->ev[3];
    cudaEvent_t main_in = side->ev[4];
    auto h2d = [&](void *dst, const void *src, size_t bytes, cudaStream_t st) {
        if (e == cudaSuccess && bytes) e = cudaMemcpyAsync(dst, src, bytes, cudaMemcpyHostToDevice, st);
    };
    auto d2h = [&](void *dst, const void *src, size_t bytes, cudaStream_t st) {
        if (e == cudaSuccess && bytes && dst) e = cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDeviceToHost, st);
    };
    // the first r columns of a T x d matrix (rows d * es bytes apart), either way: by a copy
    // kernel through the host buffer's device mapping when it has one, else a strided memcpy
    auto cols = [&](void *dst, const void *src, cudaMemcpyKind k, cudaStream_t st) {
        if (e != cudaSuccess || T == 0) return;
        const size_t pitch = (size_t)D * es, w = (size_t)r * es;
        const bool in = k == cudaMemcpyHostToDevice;
        void *mh = (w % 16 == 0 && pitch % 16 == 0 && aligned16(dst) && aligned16(src)) ? mapped_host(in ? src : dst)
                                                                                        : nullptr;
        if (!mh) {
            e = cudaMemcpy2DAsync(dst, pitch, src, pitch, w, (size_t)T, k, st);
            return;
        }
        const int64_t units = T * (int64_t)(w / 16);
        int64_t grid = (units + 255) / 256;
        if (grid > (int64_t)c.sm_count * 8) grid = (int64_t)c.sm_count * 8;
        k_copy_cols<<<(unsigned)grid, 256, 0, st>>>(static_cast<const uint4 *>(in ? mh : src),
                                                     static_cast<uint4 *>(in ? dst : mh), T, (int64_t)(pitch / 16),
                                                     (int64_t)(w / 16));
        count_launches(1);
        e = cudaGetLastError();
    };
    // inputs: what the forward reads first, on the caller's stream; then dY on the second
    // stream, travelling in while the forward runs and its results travel out
    if (a->wait_before_inputs)   // after the copies of the call that recorded it (a caller's chain)
        e = cudaStreamWaitEvent(c.stream, static_cast<cudaEvent_t>(a->wait_before_inputs), 0);
    h2d(const_cast<void *>(dv.We1), a->We1, (size_t)(D * m) * es, c.stream);
    if (!lin) h2d(const_cast<void *>(dv.We2), a->We2, (size_t)(m * r) * es, c.stream);
    if (!lin) h2d(const_cast<void *>(dv.Wd1), a->Wd1, (size_t)(r * m) * es, c.stream);
    h2d(const_cast<void *>(dv.Wd2), a->Wd2, (size_t)(m * D) * es, c.stream);
    cols(const_cast<void *>(dv.X), a->X, cudaMemcpyHostToDevice, c.stream);   // the identity path reads X[:, :r] only
    h2d(const_cast<void *>(dv.F), a->F, (size_t)(T * D) * es, c.stream);
    if (e == cudaSuccess) e = cudaEventRecord(fork, c.stream);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(s_in, fork, 0);
    h2d(const_cast<void *>(dv.dY), a->dY, (size_t)(T * D) * es, s_in);
    if (e == cudaSuccess) e = cudaEventRecord(dy_in, s_in);
    if (a->dX) cols(dv.dX, a->dX, cudaMemcpyHostToDevice, c.stream);          // the step adds dB to dX[:, :r] only
    if (a->inputs_done && e == cudaSuccess) {   // once both streams' copies in are done
        e = cudaEventRecord(main_in, c.stream);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(s_in, main_in, 0);
        if (e == cudaSuccess) e = cudaEventRecord(static_cast<cudaEvent_t>(a->inputs_done), s_in);
    }
    if (e != cudaSuccess) s = cuda_fail(e);
    // the step, the forward results leaving on the third stream while the backward runs
    if (s == RESBM_OK) s = enqueue_step(d, dv, hs.inner, c, fwd_done, dy_in);
    if (s == RESBM_OK) {
        e = cudaStreamWaitEvent(s_out, fwd_done, 0);
        d2h(a->B, dv.B, (size_t)(T * r) * es, s_out);
        d2h(a->Y, dv.Y, (size_t)(T * D) * es, s_out);
        if (e == cudaSuccess) e = cudaEventRecord(out_done, s_out);
        d2h(a->dB, dv.dB, (size_t)(T * r) * es, c.stream);
        d2h(a->dF, dv.dF, (size_t)(T * D) * es, c.stream);
        if (a->dX) cols(a->dX, dv.dX, cudaMemcpyDeviceToHost, c.stream);
        d2h(a->P, dv.P, (size_t)(T * m) * 4, c.stream);
        d2h(a->dWe1, dv.dWe1, (size_t)(D * m) * 4, c.stream);
        if (!lin) d2h(a->dWe2, dv.dWe2, (size_t)(m * r) * 4, c.stream);
        if (!lin) d2h(a->dWd1, dv.dWd1, (size_t)(r * m) * 4, c.stream);
        d2h(a->dWd2, dv.dWd2, (size_t)(m * D) * 4, c.stream);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(c.stream, out_done, 0);
        if (e != cudaSuccess) s = cuda_fail(e);
    }
    return s;
}

}  // extern "C"
