// tc.cu -- host side of the sm_103a tensor-core kernels (tcgen05 + TMA) of the ResBM boundary.
//
// All tensor-core kernels are compiled in this one translation unit (they share the device
// error word of tc_common.cuh). Tensor maps are encoded per call through the driver entry point
// cuTensorMapEncodeTiled (no link-time dependency on libcuda).
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <atomic>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <utility>

#include "tc.h"
#include "tc_common.cuh"
#include "tc_dec_fwd.cuh"
#include "tc_enc_fwd.cuh"
#include "tc_dec_bwd.cuh"
#include "tc_enc_bwd.cuh"
#include "tc_gemm.cuh"
#include "tc_spectral.cuh"
#include "tc_hbm_forms.cuh"

namespace resbm {

namespace {

PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
{
    static std::once_flag once;
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

// 2D bf16 tensor map over a row-major matrix (outer rows x inner columns, row pitch in bytes).
bool make_map(CUtensorMap *m, const void *ptr, uint64_t inner, uint64_t outer, uint64_t pitch_bytes,
              uint32_t box_inner, uint32_t box_outer, CUtensorMapSwizzle swz)
{
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {inner, outer};
    cuuint64_t strides[1] = {pitch_bytes};
    cuuint32_t box[2] = {box_inner, box_outer};
    cuuint32_t es[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr), dims, strides, box, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

CUtensorMapSwizzle swizzle_for(uint32_t row_bytes)
{
    return row_bytes == 128 ? CU_TENSOR_MAP_SWIZZLE_128B
           : row_bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                             : CU_TENSOR_MAP_SWIZZLE_32B;
}

bool al16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Every kernel of this file is launched with programmatic stream serialization: it may be
// scheduled while the previous kernel of the stream is still finishing, and waits at its start
// (griddepcontrol.wait, before touching global memory) until that kernel has completed and its
// writes are visible. What overlaps is the launch itself and the placement of CTAs on SMs that
// the previous kernel has already left.
// `cluster` > 1 launches 1-D thread-block clusters of that many CTAs (the grid is a multiple).
template <typename... KArgs, typename... Args>
cudaError_t launch_clustered(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, int cluster,
                             cudaStream_t stream, Args &&...args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cluster > 1) {
        attr[1].id = cudaLaunchAttributeClusterDimension;
        attr[1].val.clusterDim.x = (unsigned)cluster;
        attr[1].val.clusterDim.y = 1;
        attr[1].val.clusterDim.z = 1;
        cfg.numAttrs = 2;
    }
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

template <typename... KArgs, typename... Args>
cudaError_t launch(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream, Args &&...args)
{
    return launch_clustered(kernel, grid, block, smem, 1, stream, std::forward<Args>(args)...);
}

// Dynamic shared memory attribute, set once per (kernel, device): `done` is the calling
// launcher's own per-device flag array (one per kernel instantiation).
constexpr int kMaxDev = 64;
template <typename K>
cudaError_t ensure_smem(K kernel, uint32_t bytes, int dev, std::atomic<uint8_t> (&done)[kMaxDev])
{
    if (dev >= 0 && dev < kMaxDev && done[dev].load(std::memory_order_acquire)) return cudaSuccess;
    cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (e == cudaSuccess && dev >= 0 && dev < kMaxDev) done[dev].store(1, std::memory_order_release);
    return e;
}

// Number of clusters of `cl` CTAs of `kernel` (1-D, dynamic shared memory `smem`) that can be
// resident at once, asked once per (kernel, device, cluster size); `fit` is the calling
// launcher's own cache (count + 1; 0: not asked; index 0: 4 CTAs, 1: 2 CTAs). Needs the kernel's
// dynamic shared memory attribute set first. 0 if the query fails.
template <typename... KArgs>
int coresident_clusters(void (*kernel)(KArgs...), int cl, int threads, uint32_t smem, int dev,
                        std::atomic<int> (&fit)[kMaxDev][2])
{
    const int i = cl == 4 ? 0 : 1;
    const bool cached = dev >= 0 && dev < kMaxDev;
    int n = cached ? fit[dev][i].load(std::memory_order_acquire) - 1 : -1;
    if (n >= 0) return n;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)cl);
    cfg.blockDim = dim3((unsigned)threads);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)cl;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaOccupancyMaxActiveClusters(&n, kernel, &cfg) != cudaSuccess) {
        (void)cudaGetLastError();   // not an error of the caller's stream: no clusters
        n = 0;
    }
    if (cached) fit[dev][i].store(n + 1, std::memory_order_release);
    return n;
}

// Grid and cluster size of a backward launch. The persistent grid would be g_full =
// min(128-token tiles, SMs) single CTAs; clusters of 4 are taken when at least 15/16 of g_full
// CTAs fit as co-resident clusters of 4 (the grid is then that many, a multiple of 4) and each
// CTA still gets at least `min_tokens` tokens, else clusters of 2 on the same terms, else single
// CTAs. Fewer, larger weight-gradient partials cost less than the few idle SMs (these kernels
// are bound by HBM, not by SM count), but the exchange has a cost per d chunk that only a long
// enough token range per CTA hides: min_tokens is the kernel's measured crossover.
struct BwdShape {
    int grid, cl;
};
// RESBM_CLUSTER=1, 2 or 4 forces that cluster size of the backward kernels (within the
// co-residency rule above, regardless of min_tokens), and 1 runs the encoder forward as single
// CTAs instead of pairs; unset or anything else: automatic. Read at every launch.
int forced_cluster()
{
    const char *v = getenv("RESBM_CLUSTER");
    if (!v) return 0;
    const int n = atoi(v);
    return n == 1 || n == 2 || n == 4 ? n : 0;
}
int bwd_full_grid(int64_t T, int sms)
{
    int64_t g = (T + 127) / 128;
    if (g > sms) g = sms;
    return (int)(g < 1 ? 1 : g);
}
int bwd_min_grid(int64_t T, int sms)
{
    const int gf = bwd_full_grid(T, sms);
    return (15 * gf + 15) / 16;
}
// RESBM_BWD_BALANCE=0 keeps the decoder backward's grid at the cluster rule's size; unset or
// anything else: balanced (bwd_balanced). Read at every launch.
bool bwd_balance_enabled()
{
    const char *v = getenv("RESBM_BWD_BALANCE");
    return !(v && v[0] == '0' && v[1] == 0);
}
// The fewest CTAs (a multiple of cl, at most g) that leave no CTA more whole tiles than g CTAs
// do: every CTA then has the same number of tiles or one fewer, as few as possible having
// fewer. At T = 65536 (512 tiles) on 144 CTAs, 80 CTAs make a fourth tile pass while 64 are
// done after three; 128 CTAs make the same four passes each, with fewer weight-gradient
// partial slots (32 clusters instead of 36). Measured at that size (bench, two A/B pairs): the
// decoder backward 116.5 -> 115.3 us; the encoder backward 211.0 -> 214.5 us (its epilogue's
// per-tile work gains from more SMs), so only the decoder backward takes it.
int bwd_balanced(int64_t T, int g, int cl)
{
    const int64_t U = (T + 127) / 128;
    const int64_t mt = (U + g - 1) / g;                    // the most tiles a CTA gets on g CTAs
    int64_t gb = (U + mt - 1) / mt;                        // the fewest CTAs with at most mt each
    gb = (gb + cl - 1) / cl * cl;
    return gb < g ? (int)gb : g;
}
template <typename... KArgs>
BwdShape bwd_shape(void (*kernel)(KArgs...), int64_t T, int sms, int threads, uint32_t smem, int clmax,
                   int64_t min_tokens, int dev, std::atomic<int> (&fit)[kMaxDev][2], bool balance)
{
    const int gf = bwd_full_grid(T, sms);
    const int forced = forced_cluster();
    const bool bal = balance && bwd_balance_enabled();
    for (int cl = 4; cl >= 2; cl /= 2) {
        if (cl > clmax || (forced && cl != forced)) continue;
        int64_t g = (int64_t)cl * coresident_clusters(kernel, cl, threads, smem, dev, fit);
        if (g > gf) g = gf;
        g -= g % cl;
        if (g >= cl && 16 * g >= 15 * (int64_t)gf && (forced || T >= min_tokens * g))
            return BwdShape{bal ? bwd_balanced(T, (int)g, cl) : (int)g, cl};
    }
    return BwdShape{bal ? bwd_balanced(T, gf, 1) : gf, 1};
}

bool tc_width_ok(int64_t m) { return m == 16 || m == 32 || m == 64 || m == 128; }

// Persistent grid: one CTA per SM, at most one per 128-token tile (token_range).
int grid_tokens(const Ctx &c, int64_t T)
{
    int64_t g = (T + 127) / 128;
    if (g > c.sm_count) g = c.sm_count;
    return (int)(g < 1 ? 1 : g);
}

// NORM (k_dec_fwd): 0 Y; 1 Y and the row sums of squares into ss; 2 N = RMSNorm(Y) * gamma into Y
template <int M, int NORM = 0>
cudaError_t launch_dec_fwd(const resbm_desc &d, const void *B, const void *Wd1, const void *Wd2, void *Y,
                           const Ctx &c, float *ss = nullptr, const float *rstd = nullptr, const float *gamma32 = nullptr)
{
    using Cfg = tc::DecFwdCfg<M>;
    CUtensorMap m_wd2, m_y128, m_y16, m_b;
    if (!make_map(&m_wd2, Wd2, d.d, d.m, d.d * 2, 64, M, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&m_y128, Y, d.d, d.T, d.d * 2, 64, 128, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&m_y16, Y, d.d, d.T, d.d * 2, 64, 16, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&m_b, B, d.r, d.T, d.r * 2, Cfg::GB / 2, 128, swizzle_for(Cfg::GB)))
        return cudaErrorInvalidValue;
    static std::atomic<uint8_t> smem_set[kMaxDev];
    cudaError_t e = ensure_smem(tc::k_dec_fwd<M, NORM>, Cfg::SMEM_BYTES, c.device, smem_set);
    if (e != cudaSuccess) return e;
    tc::DecFwdArgs a{static_cast<const __nv_bfloat16 *>(Wd1), d.T, d.d, d.act, d.merge_identity,
                     ss, rstd, gamma32};
    // one CTA per SM, at most one per (tile, chunk) unit (the decoder forward splits tiles by columns)
    int64_t units = ((d.T + 127) / 128) * (d.d / Cfg::NCH);
    const int grid = (int)(units < c.sm_count ? (units < 1 ? 1 : units) : c.sm_count);
    e = launch(tc::k_dec_fwd<M, NORM>, grid, Cfg::THREADS, Cfg::SMEM_BYTES, c.stream, m_wd2, m_y128, m_y16,
               m_b, a);
    count_launches(1);
    return e;
}

template <int M>
cudaError_t launch_enc_fwd(const resbm_desc &d, const void *X, const void *F, const void *We1, const void *We2,
                           void *B, float *P, const Ctx &c)
{
    using Cfg = tc::EncFwdCfg<M>;
    const CUtensorMapSwizzle wswz = Cfg::WSW == 128  ? CU_TENSOR_MAP_SWIZZLE_128B
                                    : Cfg::WSW == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                                     : CU_TENSOR_MAP_SWIZZLE_32B;
    CUtensorMap m_f128, m_f16, m_we1;
    if (!make_map(&m_f128, F, d.d, d.T, d.d * 2, 64, 128, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&m_f16, F, d.d, d.T, d.d * 2, 64, 16, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&m_we1, We1, d.m, d.d, d.m * 2, Cfg::WSW / 2, 64, wswz))
        return cudaErrorInvalidValue;
    static std::atomic<uint8_t> smem_set[kMaxDev];
    cudaError_t e = ensure_smem(tc::k_enc_fwd<M>, Cfg::SMEM_BYTES, c.device, smem_set);
    if (e != cudaSuccess) return e;
    tc::EncFwdArgs a{static_cast<const __nv_bfloat16 *>(X), static_cast<const __nv_bfloat16 *>(We2),
                     static_cast<__nv_bfloat16 *>(B), P, d.T, d.d, d.act};
    // pairs of CTAs (clusters of 2), one pair per two SMs and at most one per tile, when there are
    // more tiles than SMs (single CTAs would make a second pass: the pairs split the tiles evenly)
    // and all the pairs fit at once; single CTAs otherwise (with at most one tile each they finish
    // together, and a pair's exchange of partial P costs more than its share of a tile saves:
    // T = 16384, d = 2048, 128 tiles: 22.3 us in pairs, 21.0 us single). RESBM_CLUSTER=1 forces
    // single CTAs, 2 or 4 pairs.
    const int64_t tiles = (d.T + 127) / 128;
    int cl = 1;
    int64_t grid = tiles < c.sm_count ? (tiles < 1 ? 1 : tiles) : c.sm_count;
    const int forced = forced_cluster();
    if (Cfg::SPLIT && forced != 1 && (forced != 0 || tiles > c.sm_count)) {
        static std::atomic<int> fit[kMaxDev][2];
        int64_t pairs = tiles < c.sm_count / 2 ? (tiles < 1 ? 1 : tiles) : c.sm_count / 2;
        if (pairs >= 1 && coresident_clusters(tc::k_enc_fwd<M>, 2, Cfg::THREADS, Cfg::SMEM_BYTES, c.device, fit) >= pairs) {
            cl = 2;
            grid = 2 * pairs;
        }
    }
    e = launch_clustered(tc::k_enc_fwd<M>, (unsigned)grid, Cfg::THREADS, Cfg::SMEM_BYTES, cl, c.stream, m_f128, m_f16,
                         m_we1, a);
    count_launches(1);
    return e;
}

// Scratch layout of the backward kernels: the d x m weight gradient has one fp32 slot per
// cluster (room for g_full single CTAs; tc_wgrad.cuh); the small one has one slot per (CTA, tile
// group). Every CTA has max_groups tile groups. The scratch size covers every grid the launch
// may pick (bwd_min_grid .. bwd_full_grid, and the balanced grids below them, which have no
// more tile groups per CTA and fewer CTAs), so it does not depend on the device's occupancy.
struct BwdPlan {
    int grid = 1, max_groups = 1, nch = 1;
    int64_t slots = 1;              // small partial slots
    float *part_big = nullptr;      // g_full x d x m
    float *part_small = nullptr;    // slots x small_elems
    size_t bytes = 0;
};

int bwd_max_groups(int64_t T, int grid, int nt)
{
    const int64_t U = (T + 127) / 128;   // tiles, split as token_range does
    const int64_t max_tiles = (U + grid - 1) / grid;
    const int64_t g = (max_tiles + nt - 1) / nt;
    return (int)(g < 1 ? 1 : g);
}

// grid > 0: the plan of that grid; grid == 0: the scratch size only (the largest over all grids).
BwdPlan bwd_plan(const resbm_desc &d, int sms, int grid, int nt, int64_t small_elems, void *ws)
{
    BwdPlan p;
    const int gf = bwd_full_grid(d.T, sms);
    int64_t small_slots = 0;
    if (grid > 0) {
        p.grid = grid;
        p.max_groups = bwd_max_groups(d.T, grid, nt);
        p.slots = (int64_t)grid * p.max_groups;
        small_slots = p.slots;
    } else {
        for (int g = bwd_min_grid(d.T, sms); g <= gf; ++g) {
            const int64_t s = (int64_t)g * bwd_max_groups(d.T, g, nt);
            if (s > small_slots) small_slots = s;
        }
    }
    p.nch = (int)(d.d / 128);
    WsCarver w(ws);
    p.part_big = w.take<float>((int64_t)gf * d.d * d.m);
    p.part_small = w.take<float>(small_slots * small_elems);
    p.bytes = w.used;
    return p;
}

// The two weight-gradient reductions of a backward op in one launch: the small (r x m) job
// first, on its own blocks, the large (d x m) one on the rest; one block per 32 float4 columns,
// the whole grid resident at once (8 blocks of 256 threads per SM).
const dim3 kReduceBlock(32, tc::kSlotGroups);
tc::ReduceJob reduce_job(const float *part, int64_t slots, int64_t rows, int64_t cols, float *out, int transpose,
                         int out4, int64_t cap)
{
    int64_t g = (rows * cols / 4 + 31) / 32;
    if (g > cap) g = cap;
    return tc::ReduceJob{part, slots, rows, cols, out, transpose, out4, (int)(g < 1 ? 1 : g)};
}
cudaError_t launch_reduce(const tc::ReduceJob &small, tc::ReduceJob big, const Ctx &c)
{
    const int64_t resident = (int64_t)c.sm_count * 8;
    const int64_t left = resident - small.blocks;
    if (big.blocks > left && left >= 1) big.blocks = (int)left;
    const cudaError_t e = launch(tc::k_reduce_slots, small.blocks + big.blocks, kReduceBlock, 0, c.stream, small, big);
    count_launches(1);
    return e;
}


template <int M>
cudaError_t launch_dec_bwd(const resbm_desc &d, const void *dY, const void *B, const void *Wd1, const void *Wd2,
                           void *dB, float *dWd1, float *dWd2, void *ws, const Ctx &c, bool after_independent)
{
    using Cfg = tc::DecBwdCfg<M>;
    static std::atomic<uint8_t> smem_set[kMaxDev];
    cudaError_t e = ensure_smem(tc::k_dec_bwd<M>, Cfg::SMEM_BYTES, c.device, smem_set);
    if (e != cudaSuccess) return e;
    static std::atomic<int> fit[kMaxDev][2];
    const BwdShape sh = bwd_shape(tc::k_dec_bwd<M>, d.T, c.sm_count, Cfg::THREADS, Cfg::SMEM_BYTES, Cfg::CLMAX,
                                  Cfg::CL_MIN_TOKENS, c.device, fit, true);
    const BwdPlan p = bwd_plan(d, c.sm_count, sh.grid, Cfg::NT, d.r * d.m, ws);
    CUtensorMap m_dy128, m_dy16, m_wd2, m_b, m_yr;
    if (!make_map(&m_dy128, dY, d.d, d.T, d.d * 2, 64, 128, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&m_dy16, dY, d.d, d.T, d.d * 2, 64, 16, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&m_wd2, Wd2, d.d, d.m, d.d * 2, 64, M, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&m_b, B, d.r, d.T, d.r * 2, M, 128, swizzle_for(Cfg::RB)) ||
        !make_map(&m_yr, dY, d.d, d.T, d.d * 2, M, 128, swizzle_for(Cfg::RB)))
        return cudaErrorInvalidValue;
    tc::DecBwdArgs a{static_cast<const __nv_bfloat16 *>(Wd1),
                     static_cast<__nv_bfloat16 *>(dB),
                     tc::WgradArgs{p.part_big, p.nch},
                     p.part_small, d.T, d.d, d.act, d.merge_identity, p.max_groups, after_independent ? 1 : 0};
    e = launch_clustered(tc::k_dec_bwd<M>, p.grid, Cfg::THREADS, Cfg::SMEM_BYTES, sh.cl, c.stream, m_dy128, m_dy16,
                         m_wd2, m_b, m_yr, a);
    count_launches(1);
    if (e != cudaSuccess) return e;
    // dWd2 (m x d) = sum of the per-cluster slots (d x m), transposed; dWd1 (r x m) = sum of the slices
    const int64_t cap = (int64_t)c.sm_count * 8;
    return launch_reduce(reduce_job(p.part_small, p.slots, d.r, d.m, dWd1, 0, al16(dWd1), cap),
                         reduce_job(p.part_big, p.grid / sh.cl, d.d, d.m, dWd2, 1, 0, cap), c);
}

int dec_bwd_nt(int64_t m)
{
    return m <= 16 ? tc::DecBwdCfg<16>::NT : m <= 32 ? tc::DecBwdCfg<32>::NT : tc::DecBwdCfg<64>::NT;
}

// Scratch of the encoder backward: P (T x m fp32, used when the caller has none) and the slots.
struct EncBwdWs {
    float *P;
    BwdPlan plan;
    size_t bytes;
};

// grid > 0: the plan of that grid; grid == 0: the scratch size only (bwd_plan).
EncBwdWs enc_bwd_ws(const resbm_desc &d, int sms, int grid, void *ws)
{
    EncBwdWs w{};
    WsCarver c(ws);
    w.P = c.take<float>(d.T * d.m);
    char *rest = c.take<char>(0);
    const int nt = d.m <= 16 ? tc::EncBwdCfg<16>::NT : d.m <= 32 ? tc::EncBwdCfg<32>::NT : tc::EncBwdCfg<64>::NT;
    w.plan = bwd_plan(d, sms, grid, nt, d.m * d.r, ws ? rest : nullptr);
    w.bytes = c.used + w.plan.bytes;
    return w;
}

template <int M>
cudaError_t launch_enc_bwd(const resbm_desc &d, const void *dB, const void *F, const float *P, const void *We1,
                           const void *We2, void *dF, void *dX, float *dWe1, float *dWe2, void *ws, const Ctx &c)
{
    using Cfg = tc::EncBwdCfg<M>;
    static std::atomic<uint8_t> smem_set[kMaxDev];
    cudaError_t e = ensure_smem(tc::k_enc_bwd<M>, Cfg::SMEM_BYTES, c.device, smem_set);
    if (e != cudaSuccess) return e;
    static std::atomic<int> fit[kMaxDev][2];
    const BwdShape sh = bwd_shape(tc::k_enc_bwd<M>, d.T, c.sm_count, Cfg::THREADS, Cfg::SMEM_BYTES, Cfg::CLMAX,
                                  Cfg::CL_MIN_TOKENS, c.device, fit, false);
    const EncBwdWs w = enc_bwd_ws(d, c.sm_count, sh.grid, ws);
    const BwdPlan &p = w.plan;
    CUtensorMap m_f128, m_f16, m_we1, m_df128, m_df16, m_db;
    if (!make_map(&m_f128, F, d.d, d.T, d.d * 2, 64, 128, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&m_f16, F, d.d, d.T, d.d * 2, 64, 16, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&m_we1, We1, d.m, d.d, d.m * 2, M, 128, swizzle_for(Cfg::RB)) ||
        !make_map(&m_df128, dF, d.d, d.T, d.d * 2, 64, 128, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&m_df16, dF, d.d, d.T, d.d * 2, 64, 16, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&m_db, dB, d.r, d.T, d.r * 2, M, 128, swizzle_for(Cfg::RB)))
        return cudaErrorInvalidValue;
    if (!P) {  // P = F . We1 with the forward kernel (no B), so it matches a saved P bit for bit
        e = launch_enc_fwd<M>(d, nullptr, F, We1, We2, nullptr, w.P, c);
        if (e != cudaSuccess) return e;
        P = w.P;
    }
    tc::EncBwdArgs a{P, static_cast<const __nv_bfloat16 *>(We2), static_cast<__nv_bfloat16 *>(dX),
                     tc::WgradArgs{p.part_big, p.nch}, p.part_small, d.T, d.d, d.act, p.max_groups};
    e = launch_clustered(tc::k_enc_bwd<M>, p.grid, Cfg::THREADS, Cfg::SMEM_BYTES, sh.cl, c.stream, m_f128, m_f16,
                         m_we1, m_df128, m_df16, m_db, a);
    count_launches(1);
    if (e != cudaSuccess) return e;
    const int64_t cap = (int64_t)c.sm_count * 8;
    return launch_reduce(reduce_job(p.part_small, p.slots, d.m, d.r, dWe2, 0, al16(dWe2), cap),
                         reduce_job(p.part_big, p.grid / sh.cl, d.d, d.m, dWe1, 0, al16(dWe1), cap), c);
}

// ---- the GEMM chain (tc_gemm.cuh) --------------------------------------------------------
// C = A . B with A M x K (a_mn: stored K x M row-major, else M x K) and B K x N (b_mn: stored
// K x N row-major, else N x K), all bf16 with row pitches equal to the stored widths.
int gemm_bn(int64_t N) { return N > 128 ? 256 : 128; }

// 256-row units (two 128-row MMAs sharing each B tile, GemmCfg's BM2) for 256-column products
// without a lo half, where A is K-major (measured on GB300 at d = 8192, T = 32768, m = 512:
// P = F . We1 and dQ = dY . Wd2^T 6 % and 3 % faster; the MN-major weight gradient dWe1 = F^T dP
// 6 % slower), K (per split, for a weight gradient that may split it: wg) is long enough that a
// unit's epilogue, no longer overlapped with the next unit's products, is short next to them,
// and the 256-row units still give every SM one. RESBM_GEMM_BM2 (read at every call; a tuning
// and testing knob): 0 never, 1 wherever the shape allows (either major). Both forms sum each
// output element over K in the same order; a weight gradient's split count can differ.
bool gemm_bm2(int64_t M, int64_t N, int64_t K, bool lo, bool a_mn, int sms, bool wg)
{
    if (gemm_bn(N) != 256 || lo) return false;
    const char *v = getenv("RESBM_GEMM_BM2");
    if (v && (v[0] == '0' || v[0] == '1') && v[1] == 0) return v[0] == '1';
    if (a_mn || M <= 256 || K < 2048) return false;
    int64_t units = ((M + 255) / 256) * ((N + 255) / 256);
    if (wg) units *= K / 2048 < 32 ? K / 2048 : 32;
    return units >= sms;
}

// Split-K of a product with few output tiles (the weight gradients, K = tokens): enough splits
// to give every SM a unit, at most 32 and at least four 64-deep K slices per split. rows: the
// unit's rows (256 where gemm_bm2 holds).
int gemm_splits(int64_t M, int64_t N, int64_t K, int sms, int rows = 128)
{
    const int bn = gemm_bn(N);
    const int64_t units = ((M + rows - 1) / rows) * ((N + bn - 1) / bn);
    if (4 * units >= 3 * (int64_t)sms) return 1;
    int64_t s = sms / units;
    // 256-row units keep 2048 K per split (their epilogue is not overlapped with the next unit)
    const int64_t kmax = rows == 256 ? (K / 2048 > 1 ? K / 2048 : 1) : (K + 255) / 256;
    if (s > kmax) s = kmax;
    if (s > 32) s = 32;
    if (s < 1) s = 1;
    const int64_t kc = ((K + s - 1) / s + 63) / 64 * 64;
    return (int)((K + kc - 1) / kc);
}

// MC: CTA pairs sharing B by multicast (k_gemm); the grid is then two CTAs per co-resident pair,
// at most one pair per pair unit (returns cudaErrorNotSupported, before launching, when no pair
// fits: the caller runs single CTAs).
// TS: the output leaves by TMA stores through `mo` (k_gemm's TS form); otherwise `mo` is not read.
template <int BN, bool AMN, bool BMN, bool ALO, bool ENCP = false, bool MC = false, bool BM2 = false, bool TS = false>
cudaError_t launch_gemm_t(const CUtensorMap &ma, const CUtensorMap &malo, const CUtensorMap &mb,
                          const tc::GemmShape &g, const tc::GemmEp &ep, const Ctx &c, const CUtensorMap *mo = nullptr)
{
    using Cfg = tc::GemmCfg<BN, ALO, BM2, TS>;
    const CUtensorMap &mout = mo ? *mo : ma;
#define RESBM_KGEMM tc::k_gemm<BN, AMN, BMN, ALO, ENCP, MC, BM2, TS>
    static std::atomic<uint8_t> smem_set[kMaxDev];
    cudaError_t e = ensure_smem(RESBM_KGEMM, Cfg::SMEM_BYTES, c.device, smem_set);
    if (e != cudaSuccess) return e;
    if (MC) {
        static std::atomic<int> fit[kMaxDev][2];
        const int pairs_fit = coresident_clusters(RESBM_KGEMM, 2, Cfg::THREADS,
                                                  Cfg::SMEM_BYTES, c.device, fit);
        const int64_t pair_units = (int64_t)((g.nm + 1) / 2) * g.nn * g.splits;
        const int64_t pairs = pair_units < pairs_fit ? pair_units : pairs_fit;
        if (pairs < 1) return cudaErrorNotSupported;
        e = launch_clustered(RESBM_KGEMM, (unsigned)(2 * pairs), Cfg::THREADS,
                             Cfg::SMEM_BYTES, 2, c.stream, ma, malo, mb, mout, g, ep);
    } else {
        const int64_t grid = g.units < c.sm_count ? g.units : c.sm_count;
        e = launch(RESBM_KGEMM, (unsigned)grid, Cfg::THREADS, Cfg::SMEM_BYTES, c.stream, ma,
                   malo, mb, mout, g, ep);
    }
#undef RESBM_KGEMM
    count_launches(1);
    return e;
}

// The TMA-store epilogue (k_gemm's TS form) unless RESBM_GEMM_TS=0 (read at every launch; a tuning
// and testing knob: both forms store the same bits).
bool ts_enabled()
{
    const char *v = getenv("RESBM_GEMM_TS");
    return !(v && v[0] == '0' && v[1] == 0);
}

// Pairs sharing B by multicast for the 256-column products with at least two row blocks, unless
// RESBM_GEMM_MC=0 (read at every launch; a tuning and testing knob: both forms compute the same
// bits, each output element summed in the same order by one CTA).
bool gemm_pairs(int bn, int64_t M)
{
    const char *v = getenv("RESBM_GEMM_MC");
    return bn == 256 && M > 128 && !(v && v[0] == '0' && v[1] == 0);
}

// splits: 1 for every product whose epilogue is not a plain fp32 store; with splits > 1 the
// epilogue must be GEP_F32 into `splits` slots of M x N (ep.split_stride apart). A_lo: the lo
// half of A as a bf16 hi + lo pair (same shape and layout as A), or null. rows: the unit's rows
// as the caller chose them (128 or 256), or 0 to choose here.
cudaError_t gemm(const Ctx &c, int64_t M, int64_t N, int64_t K, const void *A, bool a_mn, const void *B, bool b_mn,
                 const tc::GemmEp &ep, int splits, const void *A_lo = nullptr, int rows = 0)
{
    if (M <= 0 || N <= 0 || K <= 0) return cudaSuccess;
    const int bn = gemm_bn(N);
    CUtensorMap ma, malo, mbm;
    const bool okA = a_mn ? make_map(&ma, A, M, K, M * 2, 64, 64, CU_TENSOR_MAP_SWIZZLE_128B)
                          : make_map(&ma, A, K, M, K * 2, 64, 128, CU_TENSOR_MAP_SWIZZLE_128B);
    const bool okL = !A_lo ? true
                     : a_mn ? make_map(&malo, A_lo, M, K, M * 2, 64, 64, CU_TENSOR_MAP_SWIZZLE_128B)
                            : make_map(&malo, A_lo, K, M, K * 2, 64, 128, CU_TENSOR_MAP_SWIZZLE_128B);
    const bool lo = A_lo != nullptr;
    const bool bm2 = !lo && bn == 256 && (rows ? rows == 256 : gemm_bm2(M, N, K, lo, a_mn, c.sm_count, false));
    const bool pair = !bm2 && gemm_pairs(bn, M);
    // K-major B: a pair's CTAs each load half of the B tile's rows
    const bool okB = b_mn ? make_map(&mbm, B, N, K, N * 2, 64, 64, CU_TENSOR_MAP_SWIZZLE_128B)
                          : make_map(&mbm, B, K, N, K * 2, 64, (uint32_t)(pair ? bn / 2 : bn), CU_TENSOR_MAP_SWIZZLE_128B);
    if (!okA || !okL || !okB) return cudaErrorInvalidValue;
    if (!A_lo) malo = ma;   // not read
    tc::GemmShape g;
    g.M = M;
    g.N = N;
    g.K = K;
    g.splits = splits < 1 ? 1 : splits;
    g.kc = ((K + g.splits - 1) / g.splits + 63) / 64 * 64;
    g.splits = (int)((K + g.kc - 1) / g.kc);
    g.nm = (int)(bm2 ? (M + 255) / 256 : (M + 127) / 128);
    g.nn = (int)((N + bn - 1) / bn);
    g.units = (int64_t)g.nm * g.nn * g.splits;
    if (bm2) {
        if (!a_mn && b_mn) return launch_gemm_t<256, false, true, false, false, false, true>(ma, malo, mbm, g, ep, c);
        if (!a_mn && !b_mn) return launch_gemm_t<256, false, false, false, false, false, true>(ma, malo, mbm, g, ep, c);
        if (a_mn && b_mn) return launch_gemm_t<256, true, true, false, false, false, true>(ma, malo, mbm, g, ep, c);
        return cudaErrorNotSupported;
    }
    // TMA-store epilogue for the pairs' plain bf16 outputs (Y = G . Wd2 + pad(B), dF = dP . We1^T)
    CUtensorMap mo;
    const bool ts = bn == 256 && !bm2 && !a_mn && !(b_mn && lo) && g.splits == 1 &&
                    (ep.mode == tc::GEP_BF16 || ep.mode == tc::GEP_ADD_AUX || ep.mode == tc::GEP_DF) &&
                    al16(ep.out) && (ep.ldo * 2) % 16 == 0 && ts_enabled() &&
                    make_map(&mo, ep.out, N, M, ep.ldo * 2, 64, 128, CU_TENSOR_MAP_SWIZZLE_128B);
    if (ts && pair) {
        cudaError_t e = b_mn ? launch_gemm_t<256, false, true, false, false, true, false, true>(ma, malo, mbm, g, ep, c, &mo)
                        : lo ? launch_gemm_t<256, false, false, true, false, true, false, true>(ma, malo, mbm, g, ep, c, &mo)
                             : launch_gemm_t<256, false, false, false, false, true, false, true>(ma, malo, mbm, g, ep, c, &mo);
        if (e != cudaErrorNotSupported) return e;
        // no pair fits: single CTAs need the whole-tile box for K-major B
        if (!b_mn && !make_map(&mbm, B, K, N, K * 2, 64, (uint32_t)bn, CU_TENSOR_MAP_SWIZZLE_128B))
            return cudaErrorInvalidValue;
    }
    if (ts) {   // single CTAs
        return b_mn ? launch_gemm_t<256, false, true, false, false, false, false, true>(ma, malo, mbm, g, ep, c, &mo)
               : lo ? launch_gemm_t<256, false, false, true, false, false, false, true>(ma, malo, mbm, g, ep, c, &mo)
                    : launch_gemm_t<256, false, false, false, false, false, false, true>(ma, malo, mbm, g, ep, c, &mo);
    }
    if (pair) {
        cudaError_t e = cudaErrorNotSupported;
        if (!a_mn && b_mn) e = lo ? launch_gemm_t<256, false, true, true, false, true>(ma, malo, mbm, g, ep, c)
                                  : launch_gemm_t<256, false, true, false, false, true>(ma, malo, mbm, g, ep, c);
        else if (!a_mn && !b_mn) e = lo ? launch_gemm_t<256, false, false, true, false, true>(ma, malo, mbm, g, ep, c)
                                        : launch_gemm_t<256, false, false, false, false, true>(ma, malo, mbm, g, ep, c);
        else if (a_mn && b_mn) e = lo ? launch_gemm_t<256, true, true, true, false, true>(ma, malo, mbm, g, ep, c)
                                      : launch_gemm_t<256, true, true, false, false, true>(ma, malo, mbm, g, ep, c);
        if (e != cudaErrorNotSupported) return e;
        // no pair fits: single CTAs need the whole-tile box for K-major B
        if (!b_mn && !make_map(&mbm, B, K, N, K * 2, 64, (uint32_t)bn, CU_TENSOR_MAP_SWIZZLE_128B))
            return cudaErrorInvalidValue;
    }
    if (bn == 256) {
        if (!a_mn && b_mn) return lo ? launch_gemm_t<256, false, true, true>(ma, malo, mbm, g, ep, c)
                                     : launch_gemm_t<256, false, true, false>(ma, malo, mbm, g, ep, c);
        if (!a_mn && !b_mn) return lo ? launch_gemm_t<256, false, false, true>(ma, malo, mbm, g, ep, c)
                                      : launch_gemm_t<256, false, false, false>(ma, malo, mbm, g, ep, c);
        if (a_mn && b_mn) return lo ? launch_gemm_t<256, true, true, true>(ma, malo, mbm, g, ep, c)
                                    : launch_gemm_t<256, true, true, false>(ma, malo, mbm, g, ep, c);
    } else {
        if (!a_mn && b_mn) return lo ? launch_gemm_t<128, false, true, true>(ma, malo, mbm, g, ep, c)
                                     : launch_gemm_t<128, false, true, false>(ma, malo, mbm, g, ep, c);
        if (!a_mn && !b_mn) return lo ? launch_gemm_t<128, false, false, true>(ma, malo, mbm, g, ep, c)
                                      : launch_gemm_t<128, false, false, false>(ma, malo, mbm, g, ep, c);
        if (a_mn && b_mn) return lo ? launch_gemm_t<128, true, true, true>(ma, malo, mbm, g, ep, c)
                                    : launch_gemm_t<128, true, true, false>(ma, malo, mbm, g, ep, c);
    }
    return cudaErrorNotSupported;
}

tc::GemmEp ep_of(int mode, int act, void *out, int64_t ldo)
{
    tc::GemmEp e{};
    e.mode = mode;
    e.act = act;
    e.out = out;
    e.ldo = ldo;
    return e;
}

// A weight gradient W (M x N fp32) = A^T . B over K tokens (both operands MN-major), split over
// the tokens when it has few output tiles: the splits' fp32 slots go to `slots` and the job to
// sum them (in slot order) is returned in `job` (job->blocks = 0: nothing to reduce).
// A_lo: A as a bf16 hi + lo pair (or null). a_mn / b_mn: the operand majors (both MN-major for the
// weight gradients, whose K is the tokens).
cudaError_t wgrad(const Ctx &c, int64_t M, int64_t N, int64_t K, const void *A, const void *B, float *W, float *slots,
                  tc::ReduceJob *job, const void *A_lo = nullptr, bool a_mn = true, bool b_mn = true)
{
    const int rows = gemm_bm2(M, N, K, A_lo != nullptr, a_mn, c.sm_count, true) ? 256 : 128;
    const int s = gemm_splits(M, N, K, c.sm_count, rows);
    *job = tc::ReduceJob{nullptr, 0, 0, 0, nullptr, 0, 0, 0};
    if (s <= 1) return gemm(c, M, N, K, A, a_mn, B, b_mn, ep_of(tc::GEP_F32, 0, W, N), 1, A_lo, rows);
    tc::GemmEp e = ep_of(tc::GEP_F32, 0, slots, N);
    e.split_stride = M * N;
    cudaError_t err = gemm(c, M, N, K, A, a_mn, B, b_mn, e, s, A_lo, rows);
    if (err != cudaSuccess) return err;
    // the number of splits the launch took (gemm rounds K per split to 64)
    const int64_t kc = ((K + s - 1) / s + 63) / 64 * 64;
    const int64_t ns = (K + kc - 1) / kc;
    *job = reduce_job(slots, ns, M, N, W, 0, al16(W), (int64_t)c.sm_count * 8);
    return cudaSuccess;
}

cudaError_t reduce_jobs(const tc::ReduceJob &a, const tc::ReduceJob &b, const Ctx &c)
{
    if (a.blocks == 0 && b.blocks == 0) return cudaSuccess;
    const tc::ReduceJob none{nullptr, 0, 0, 0, nullptr, 0, 0, 0};
    const tc::ReduceJob &first = a.blocks ? a : none;
    const tc::ReduceJob &second = a.blocks ? (b.blocks ? b : none) : b;
    const int blocks = first.blocks + second.blocks;
    const cudaError_t e = launch(tc::k_reduce_slots, blocks, kReduceBlock, 0, c.stream, first, second);
    count_launches(1);
    return e;
}

// Scratch of the GEMM chain of each op (grid == the device's SMs): the intermediate T x m
// tensors and the weight gradients' split slots.
struct GemmWs {
    float *P = nullptr, *Q = nullptr;
    __nv_bfloat16 *A = nullptr, *G = nullptr, *dQ = nullptr, *dP = nullptr;
    __nv_bfloat16 *A_lo = nullptr, *G_lo = nullptr, *dQ_lo = nullptr, *dP_lo = nullptr;   // remainders of hi + lo pairs
    float *slots1 = nullptr, *slots2 = nullptr;
    size_t bytes = 0;
};

// dF = dP . We1^T takes dP as a hi + lo pair up to this hidden width (K = m is short there and
// the product is bound by the dF stream; at larger m it would double the op's largest product)
constexpr int64_t kDfLoMaxM = 64;

size_t slot_floats(int64_t M, int64_t N, int64_t K, int sms)
{
    // room for either unit size (which one a launch takes can depend on RESBM_GEMM_BM2)
    const int s1 = gemm_splits(M, N, K, sms, 128), s2 = gemm_splits(M, N, K, sms, 256);
    const int s = s1 > s2 ? s1 : s2;
    return s > 1 ? (size_t)(s * M * N) : 0;
}

GemmWs gemm_ws(const resbm_desc &d, int op, int sms, void *ws, bool have_P)
{
    GemmWs w;
    WsCarver cv(ws);
    const int64_t T = d.T, D = d.d, r = d.r, m = d.m;
    if (op == RESBM_OP_ENCODE_FWD) {
        w.A = cv.take<__nv_bfloat16>(T * m);
        w.A_lo = cv.take<__nv_bfloat16>(T * m);
    } else if (op == RESBM_OP_DECODE_FWD) {
        w.G = cv.take<__nv_bfloat16>(T * m);
    } else if (op == RESBM_OP_DECODE_BWD) {
        w.Q = cv.take<float>(T * m);
        w.G = cv.take<__nv_bfloat16>(T * m);
        w.G_lo = cv.take<__nv_bfloat16>(T * m);
        w.dQ = cv.take<__nv_bfloat16>(T * m);
        w.dQ_lo = cv.take<__nv_bfloat16>(T * m);
        w.slots1 = cv.take<float>(slot_floats(m, D, T, sms));   // dWd2
        w.slots2 = cv.take<float>(slot_floats(r, m, T, sms));   // dWd1
    } else if (op == RESBM_OP_ENCODE_BWD) {
        if (!have_P) w.P = cv.take<float>(T * m);
        w.A = cv.take<__nv_bfloat16>(T * m);
        w.dP = cv.take<__nv_bfloat16>(T * m);
        if (m <= kDfLoMaxM) w.dP_lo = cv.take<__nv_bfloat16>(T * m);
        w.slots1 = cv.take<float>(slot_floats(D, m, T, sms));   // dWe1
        w.slots2 = cv.take<float>(slot_floats(m, r, T, sms));   // dWe2
    }
    w.bytes = cv.used;
    return w;
}

}  // namespace

bool tc_supported(const resbm_desc &d, int op)
{
    if (d.dtype != RESBM_BF16 || d.m != d.r || !tc_width_ok(d.m)) return false;
    if (d.T > INT32_MAX || encode_fn() == nullptr) return false;
    if (op == RESBM_OP_DECODE_FWD) {
        const int64_t nch = d.m <= 32 ? 256 : 128;
        return d.d % nch == 0;
    }
    if (op == RESBM_OP_ENCODE_FWD) return d.d % 64 == 0;
    if (op == RESBM_OP_DECODE_BWD || op == RESBM_OP_ENCODE_BWD) return d.m <= 64 && d.d % 128 == 0;
    return false;
}

size_t tc_ws_bytes(const resbm_desc &d, int op, int sms)
{
    if (op == RESBM_OP_DECODE_BWD) return bwd_plan(d, sms, 0, dec_bwd_nt(d.m), d.r * d.m, nullptr).bytes;
    if (op == RESBM_OP_ENCODE_BWD) return enc_bwd_ws(d, sms, 0, nullptr).bytes;
    return 0;
}

cudaError_t tc_encode_fwd(const resbm_desc &d, const void *X, const void *F, const void *We1, const void *We2,
                          void *B, float *P, void *, const Ctx &c)
{
    if (!al16(X) || !al16(F) || !al16(We1) || !al16(We2) || !al16(B) || (P && !al16(P)))
        return cudaErrorNotSupported;
    switch (d.m) {
    case 16: return launch_enc_fwd<16>(d, X, F, We1, We2, B, P, c);
    case 32: return launch_enc_fwd<32>(d, X, F, We1, We2, B, P, c);
    case 64: return launch_enc_fwd<64>(d, X, F, We1, We2, B, P, c);
    case 128: return launch_enc_fwd<128>(d, X, F, We1, We2, B, P, c);
    }
    return cudaErrorNotSupported;
}

cudaError_t tc_decode_fwd(const resbm_desc &d, const void *B, const void *Wd1, const void *Wd2, void *Y, void *,
                          const Ctx &c)
{
    if (!al16(B) || !al16(Wd1) || !al16(Wd2) || !al16(Y)) return cudaErrorNotSupported;
    switch (d.m) {
    case 16: return launch_dec_fwd<16>(d, B, Wd1, Wd2, Y, c);
    case 32: return launch_dec_fwd<32>(d, B, Wd1, Wd2, Y, c);
    case 64: return launch_dec_fwd<64>(d, B, Wd1, Wd2, Y, c);
    case 128: return launch_dec_fwd<128>(d, B, Wd1, Wd2, Y, c);
    }
    return cudaErrorNotSupported;
}

// gamma as fp32 (d), the row sums of squares (2 d / NCH slots of T), the T reciprocal RMS values
int rmsnorm_slots(const resbm_desc &d) { return (int)(2 * (d.d / (d.m <= 32 ? 256 : 128))); }   // NCH
size_t tc_rmsnorm_ws_bytes(const resbm_desc &d)
{
    return ((size_t)d.d + ((size_t)rmsnorm_slots(d) + 1) * (size_t)d.T) * sizeof(float);
}

template <int M>
cudaError_t dec_fwd_rmsnorm_t(const resbm_desc &d, const void *B, const void *Wd1, const void *Wd2,
                              const void *gamma, float eps, void *Y, void *N, float *ss, const Ctx &c)
{
    static_assert(tc::DecFwdCfg<M>::NCH == (M <= 32 ? 256 : 128), "rmsnorm_slots");
    const int ns = rmsnorm_slots(d);
    float *gamma32 = ss;   // first: d floats, a multiple of NCH, so the slots stay 16-byte aligned too
    ss += d.d;
    float *rstd = ss + (int64_t)ns * d.T;
    cudaError_t e = launch_dec_fwd<M, 1>(d, B, Wd1, Wd2, Y, c, ss);
    if (e != cudaSuccess) return e;
    const int64_t n = d.T > d.d ? d.T : d.d;
    int64_t blocks = (n + 255) / 256;
    if (blocks > (int64_t)c.sm_count * 8) blocks = (int64_t)c.sm_count * 8;
    e = launch(tc::k_row_rstd, (unsigned)blocks, 256, 0, c.stream, (const float *)ss, ns, d.T, d.d, eps, rstd,
               static_cast<const __nv_bfloat16 *>(gamma), gamma32);
    count_launches(1);
    return e != cudaSuccess ? e : launch_dec_fwd<M, 2>(d, B, Wd1, Wd2, N, c, nullptr, rstd, gamma32);
}

cudaError_t tc_decode_fwd_rmsnorm(const resbm_desc &d, const void *B, const void *Wd1, const void *Wd2,
                                  const void *gamma, float eps, void *Y, void *N, void *ws, const Ctx &c)
{
    if (!al16(B) || !al16(Wd1) || !al16(Wd2) || !al16(Y) || !al16(N) || !al16(ws))
        return cudaErrorNotSupported;
    float *ss = static_cast<float *>(ws);
    switch (d.m) {
    case 16: return dec_fwd_rmsnorm_t<16>(d, B, Wd1, Wd2, gamma, eps, Y, N, ss, c);
    case 32: return dec_fwd_rmsnorm_t<32>(d, B, Wd1, Wd2, gamma, eps, Y, N, ss, c);
    case 64: return dec_fwd_rmsnorm_t<64>(d, B, Wd1, Wd2, gamma, eps, Y, N, ss, c);
    case 128: return dec_fwd_rmsnorm_t<128>(d, B, Wd1, Wd2, gamma, eps, Y, N, ss, c);
    }
    return cudaErrorNotSupported;
}

cudaError_t tc_decode_bwd(const resbm_desc &d, const void *dY, const void *B, const void *Wd1, const void *Wd2,
                          void *dB, float *dWd1, float *dWd2, void *ws, const Ctx &c, bool after_independent)
{
    if (!al16(dY) || !al16(B) || !al16(Wd1) || !al16(Wd2) || !al16(dB)) return cudaErrorNotSupported;
    switch (d.m) {
    case 16: return launch_dec_bwd<16>(d, dY, B, Wd1, Wd2, dB, dWd1, dWd2, ws, c, after_independent);
    case 32: return launch_dec_bwd<32>(d, dY, B, Wd1, Wd2, dB, dWd1, dWd2, ws, c, after_independent);
    case 64: return launch_dec_bwd<64>(d, dY, B, Wd1, Wd2, dB, dWd1, dWd2, ws, c, after_independent);
    }
    return cudaErrorNotSupported;
}

cudaError_t tc_encode_bwd(const resbm_desc &d, const void *dB, const void *F, const float *P, const void *We1,
                          const void *We2, void *dF, void *dX, float *dWe1, float *dWe2, void *ws, const Ctx &c)
{
    if (!al16(dB) || !al16(F) || (P && !al16(P)) || !al16(We1) || !al16(We2) || !al16(dF) || (dX && !al16(dX)))
        return cudaErrorNotSupported;
    switch (d.m) {
    case 16: return launch_enc_bwd<16>(d, dB, F, P, We1, We2, dF, dX, dWe1, dWe2, ws, c);
    case 32: return launch_enc_bwd<32>(d, dB, F, P, We1, We2, dF, dX, dWe1, dWe2, ws, c);
    case 64: return launch_enc_bwd<64>(d, dB, F, P, We1, We2, dF, dX, dWe1, dWe2, ws, c);
    }
    return cudaErrorNotSupported;
}

// ---- the GEMM chain of each op ------------------------------------------------------------
bool gemm_supported(const resbm_desc &d, int op)
{
    if (d.dtype != RESBM_BF16 || d.T > INT32_MAX || encode_fn() == nullptr) return false;
    if (d.d % 8 || d.r % 8 || d.m % 8) return false;   // 16-byte row pitches (TMA, vector epilogues)
    return op >= RESBM_OP_ENCODE_FWD && op <= RESBM_OP_ENCODE_BWD;
}

size_t gemm_ws_bytes(const resbm_desc &d, int op, int sms) { return gemm_ws(d, op, sms, nullptr, false).bytes; }

cudaError_t gemm_encode_fwd(const resbm_desc &d, const void *X, const void *F, const void *We1, const void *We2,
                            void *B, float *P, void *ws, const Ctx &c)
{
    if (!al16(X) || !al16(F) || !al16(We1) || !al16(We2) || !al16(B) || (P && !al16(P)) || !al16(ws))
        return cudaErrorNotSupported;
    const GemmWs w = gemm_ws(d, RESBM_OP_ENCODE_FWD, c.sm_count, ws, true);
    // P = F . We1 (saved if asked), A = phi(P)
    tc::GemmEp e1 = ep_of(tc::GEP_P_A, d.act, P, d.m);
    e1.out2 = w.A;
    e1.ldo2 = d.m;
    e1.lo = w.A_lo;
    cudaError_t e = gemm(c, d.T, d.m, d.d, F, false, We1, true, e1, 1);
    if (e != cudaSuccess) return e;
    // B = X[:, :r] + (A_hi + A_lo) . We2 (the truncating identity path added in the epilogue)
    tc::GemmEp e2 = ep_of(tc::GEP_ADD_AUX, d.act, B, d.r);
    e2.aux = X;
    e2.lda = d.d;
    e2.aux_cols = d.r;
    return gemm(c, d.T, d.r, d.m, w.A, false, We2, true, e2, 1, w.A_lo);
}

cudaError_t gemm_decode_fwd(const resbm_desc &d, const void *B, const void *Wd1, const void *Wd2, void *Y, void *ws,
                            const Ctx &c)
{
    if (!al16(B) || !al16(Wd1) || !al16(Wd2) || !al16(Y) || !al16(ws)) return cudaErrorNotSupported;
    const GemmWs w = gemm_ws(d, RESBM_OP_DECODE_FWD, c.sm_count, ws, true);
    // G = phi(B . Wd1)
    cudaError_t e = gemm(c, d.T, d.m, d.r, B, false, Wd1, true, ep_of(tc::GEP_ACT, d.act, w.G, d.m), 1);
    if (e != cudaSuccess) return e;
    // Y = G . Wd2 (+ B on the first r columns: the zero-padding identity path)
    tc::GemmEp e2 = ep_of(tc::GEP_ADD_AUX, d.act, Y, d.d);
    e2.aux = d.merge_identity ? B : nullptr;
    e2.lda = d.r;
    e2.aux_cols = d.merge_identity ? d.r : 0;
    return gemm(c, d.T, d.d, d.m, w.G, false, Wd2, true, e2, 1);
}

cudaError_t gemm_decode_bwd(const resbm_desc &d, const void *dY, const void *B, const void *Wd1, const void *Wd2,
                            void *dB, float *dWd1, float *dWd2, void *ws, const Ctx &c)
{
    if (!al16(dY) || !al16(B) || !al16(Wd1) || !al16(Wd2) || !al16(dB) || !al16(dWd1) || !al16(dWd2) || !al16(ws))
        return cudaErrorNotSupported;
    const GemmWs w = gemm_ws(d, RESBM_OP_DECODE_BWD, c.sm_count, ws, true);
    // Q = B . Wd1 (kept), G = phi(Q) as a hi + lo pair
    tc::GemmEp e1 = ep_of(tc::GEP_ACT, d.act, w.G, d.m);
    e1.out2 = w.Q;
    e1.ldo2 = d.m;
    e1.lo = w.G_lo;
    cudaError_t e = gemm(c, d.T, d.m, d.r, B, false, Wd1, true, e1, 1);
    // dQ = (dY . Wd2^T) * phi'(Q)
    tc::GemmEp e2 = ep_of(tc::GEP_DACT, d.act, w.dQ, d.m);
    e2.aux = w.Q;
    e2.lda = d.m;
    e2.lo = w.dQ_lo;
    if (e == cudaSuccess) e = gemm(c, d.T, d.m, d.d, dY, false, Wd2, false, e2, 1);
    // dB = [merge] dY[:, :r] + (dQ_hi + dQ_lo) . Wd1^T
    tc::GemmEp e3 = ep_of(tc::GEP_ADD_AUX, d.act, dB, d.r);
    e3.aux = d.merge_identity ? dY : nullptr;
    e3.lda = d.d;
    e3.aux_cols = d.merge_identity ? d.r : 0;
    if (e == cudaSuccess) e = gemm(c, d.T, d.r, d.m, w.dQ, false, Wd1, false, e3, 1, w.dQ_lo);
    // dWd2 = (G_hi + G_lo)^T . dY, dWd1 = B^T . dQ (sums over the tokens)
    tc::ReduceJob j2, j1;
    if (e == cudaSuccess) e = wgrad(c, d.m, d.d, d.T, w.G, dY, dWd2, w.slots1, &j2, w.G_lo);
    if (e == cudaSuccess) e = wgrad(c, d.r, d.m, d.T, B, w.dQ, dWd1, w.slots2, &j1);
    if (e == cudaSuccess) e = reduce_jobs(j1, j2, c);
    return e;
}

cudaError_t gemm_encode_bwd(const resbm_desc &d, const void *dB, const void *F, const float *P, const void *We1,
                            const void *We2, void *dF, void *dX, float *dWe1, float *dWe2, void *ws, const Ctx &c)
{
    if (!al16(dB) || !al16(F) || (P && !al16(P)) || !al16(We1) || !al16(We2) || !al16(dF) || (dX && !al16(dX)) ||
        !al16(dWe1) || !al16(dWe2) || !al16(ws))
        return cudaErrorNotSupported;
    const GemmWs w = gemm_ws(d, RESBM_OP_ENCODE_BWD, c.sm_count, ws, P != nullptr);
    cudaError_t e = cudaSuccess;
    if (!P) {   // P = F . We1, the forward's own product (the same launch shape, so the same bits)
        tc::GemmEp e0 = ep_of(tc::GEP_P_A, d.act, w.P, d.m);
        e0.out2 = w.A;   // overwritten below; the forward writes A too
        e0.ldo2 = d.m;
        e = gemm(c, d.T, d.m, d.d, F, false, We1, true, e0, 1);
        P = w.P;
    }
    // dP = (dB . We2^T) * phi'(P), and A = phi(P) for dWe2
    tc::GemmEp e1 = ep_of(tc::GEP_DACT, d.act, w.dP, d.m);
    e1.aux = P;
    e1.lda = d.m;
    e1.out2 = w.A;
    e1.ldo2 = d.m;
    e1.lo = w.dP_lo;
    if (e == cudaSuccess) e = gemm(c, d.T, d.m, d.r, dB, false, We2, false, e1, 1);
    // dF = dP . We1^T (dP as a hi + lo pair at small m), and dX[:, :r] += dB (the gradient of
    // the truncating identity path)
    tc::GemmEp e2 = ep_of(tc::GEP_DF, d.act, dF, d.d);
    e2.rmw = static_cast<__nv_bfloat16 *>(dX);
    e2.ldr = d.d;
    e2.aux = dB;
    e2.lda = d.r;
    e2.aux_cols = d.r;
    if (e == cudaSuccess) e = gemm(c, d.T, d.d, d.m, w.dP, false, We1, false, e2, 1, w.dP_lo);
    // dWe1 = F^T . dP, dWe2 = A^T . dB
    tc::ReduceJob j1, j2;
    if (e == cudaSuccess) e = wgrad(c, d.d, d.m, d.T, F, w.dP, dWe1, w.slots1, &j1);
    if (e == cudaSuccess) e = wgrad(c, d.m, d.r, d.T, w.A, dB, dWe2, w.slots2, &j2);
    if (e == cudaSuccess) e = reduce_jobs(j2, j1, c);
    return e;
}

// ---- the encoder fused into the FFN down-projection ---------------------------------------------
namespace {
int ffn_bn(int64_t d) { return d > 128 ? 256 : 128; }
int64_t ffn_slots(const resbm_desc &d) { return 2 * ((d.d + ffn_bn(d.d) - 1) / ffn_bn(d.d)); }
}  // namespace

bool ffn_encode_supported(const resbm_desc &d, int64_t f)
{
    return d.dtype == RESBM_BF16 && !(d.flags & RESBM_FLAG_LINEAR) && d.m % 8 == 0 && d.m <= 32 && d.r <= 32 &&
           d.d % 8 == 0 && f >= 1 && f % 8 == 0 && d.T <= INT32_MAX;
}

size_t ffn_encode_ws_bytes(const resbm_desc &d, int64_t f)
{
    (void)f;
    WsCarver cv(nullptr);
    cv.take<float>(ffn_slots(d) * d.T * d.m);
    return cv.used;
}

cudaError_t tc_ffn_down_encode(const resbm_desc &d, int64_t f, const void *H, const void *W2, const void *X,
                               const void *We1, const void *We2, void *B, float *P, void *F_out, void *ws,
                               const Ctx &c)
{
    if (!al16(H) || !al16(W2) || !al16(We1) || !al16(ws) || (F_out && !al16(F_out)) || (P && !al16(P)) ||
        encode_fn() == nullptr)
        return cudaErrorNotSupported;
    const int bn = ffn_bn(d.d);
    CUtensorMap ma, mb;
    if (!make_map(&ma, H, f, d.T, f * 2, 64, 128, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&mb, W2, d.d, f, d.d * 2, 64, 64, CU_TENSOR_MAP_SWIZZLE_128B))
        return cudaErrorInvalidValue;
    tc::GemmShape g;
    g.M = d.T;
    g.N = d.d;
    g.K = f;
    g.splits = 1;
    g.kc = (f + 63) / 64 * 64;
    g.nm = (int)((d.T + 127) / 128);
    g.nn = (int)((d.d + bn - 1) / bn);
    g.units = (int64_t)g.nm * g.nn;
    tc::GemmEp e{};
    e.out = F_out;
    e.ldo = d.d;
    e.we1 = static_cast<const __nv_bfloat16 *>(We1);
    e.pslots = static_cast<float *>(ws);
    e.slot_stride = d.T * d.m;
    e.pm = (int)d.m;
    cudaError_t err = cudaErrorNotSupported;
    // (not in 256-row units: measured 0.31 -> 0.47 ms at T = 16384, f = 5632, d = 2048, the P
    // partials' epilogue no longer hidden behind the next unit's products)
    if (gemm_pairs(bn, d.T)) err = launch_gemm_t<256, false, true, false, true, true>(ma, ma, mb, g, e, c);
    if (err == cudaErrorNotSupported)
        err = bn == 256 ? launch_gemm_t<256, false, true, false, true>(ma, ma, mb, g, e, c)
                        : launch_gemm_t<128, false, true, false, true>(ma, ma, mb, g, e, c);
    if (err != cudaSuccess) return err;
    err = launch(tc::k_enc_finish, (unsigned)((d.T + 7) / 8), 256, 0, c.stream, (const float *)ws,
                 (int)ffn_slots(d), d.T * d.m, d.T, (int)d.m, (int)d.r, d.act, P,
                 static_cast<const __nv_bfloat16 *>(We2), static_cast<const __nv_bfloat16 *>(X), d.d,
                 static_cast<__nv_bfloat16 *>(B));
    count_launches(1);
    return err;
}

// ---- Muon's Newton-Schulz orthogonalisation and the effective rank ----------------------------
namespace {
// Scratch: the sum-of-squares partials, the two bf16 iterates (or the Gram matrix and its split
// slots for the effective rank), and the s x s products (s = min(rows, cols)).
struct MatrixWs {
    double *part = nullptr;
    __nv_bfloat16 *X = nullptr, *A = nullptr, *Bm = nullptr;
    float *gram = nullptr, *slots = nullptr;
    double *out = nullptr;
    size_t bytes = 0;
};
MatrixWs matrix_ws(int op, int64_t rows, int64_t cols, int sms, void *ws)
{
    MatrixWs w;
    WsCarver cv(ws);
    const int64_t sd = rows < cols ? rows : cols, ld = rows < cols ? cols : rows;
    if (op == RESBM_OP_NEWTON_SCHULZ) {
        w.part = cv.take<double>(tc::kSqBlocks);
        w.X = cv.take<__nv_bfloat16>(rows * cols);
        w.A = cv.take<__nv_bfloat16>(sd * sd);
        w.Bm = cv.take<__nv_bfloat16>(sd * sd);
    } else {
        w.gram = cv.take<float>(sd * sd);
        w.slots = cv.take<float>(slot_floats(sd, sd, ld, sms));
    }
    w.bytes = cv.used;
    return w;
}
}  // namespace

size_t matrix_ws_bytes(int op, int64_t rows, int64_t cols, int sms) { return matrix_ws(op, rows, cols, sms, nullptr).bytes; }

bool matrix_supported(int64_t rows, int64_t cols)
{
    return rows >= 1 && cols >= 1 && rows % 8 == 0 && cols % 8 == 0 && rows <= INT32_MAX && cols <= INT32_MAX;
}

cudaError_t tc_newton_schulz(int64_t rows, int64_t cols, const void *G, bool g_f32, int steps, const float coef[3],
                             float eps, void *X_out, void *ws, const Ctx &c)
{
    if (!al16(G) || !al16(X_out) || !al16(ws) || encode_fn() == nullptr) return cudaErrorNotSupported;
    const MatrixWs w = matrix_ws(RESBM_OP_NEWTON_SCHULZ, rows, cols, c.sm_count, ws);
    const int64_t n = rows * cols;
    __nv_bfloat16 *out = static_cast<__nv_bfloat16 *>(X_out);
    // the iterates alternate between the output and the scratch copy so that the last one lands in
    // the output: X0 in the scratch copy for an odd number of steps
    __nv_bfloat16 *cur = steps % 2 ? w.X : out, *nxt = steps % 2 ? out : w.X;
    int64_t grid = (n + 255) / 256;
    if (grid > (int64_t)c.sm_count * 8) grid = (int64_t)c.sm_count * 8;
    cudaError_t e;
    if (g_f32) {
        e = launch(tc::k_sumsq<float>, tc::kSqBlocks, 256, 0, c.stream, static_cast<const float *>(G), n, w.part);
        if (e == cudaSuccess)
            e = launch(tc::k_scale_bf16<float>, (unsigned)grid, 256, 0, c.stream, static_cast<const float *>(G), n,
                       (const double *)w.part, eps, cur);
    } else {
        e = launch(tc::k_sumsq<__nv_bfloat16>, tc::kSqBlocks, 256, 0, c.stream, static_cast<const __nv_bfloat16 *>(G),
                   n, w.part);
        if (e == cudaSuccess)
            e = launch(tc::k_scale_bf16<__nv_bfloat16>, (unsigned)grid, 256, 0, c.stream,
                       static_cast<const __nv_bfloat16 *>(G), n, (const double *)w.part, eps, cur);
    }
    count_launches(2);
    const bool wide = rows <= cols;
    const int64_t sd = wide ? rows : cols;
    for (int k = 0; k < steps && e == cudaSuccess; ++k) {
        // A = X X^T (wide) or X^T X (tall): the s x s Gram matrix of the iterate
        e = wide ? gemm(c, sd, sd, cols, cur, false, cur, false, ep_of(tc::GEP_BF16, 0, w.A, sd), 1)
                 : gemm(c, sd, sd, rows, cur, true, cur, true, ep_of(tc::GEP_BF16, 0, w.A, sd), 1);
        // Bm = b A + c A A
        tc::GemmEp eb = ep_of(tc::GEP_AXPBY, 0, w.Bm, sd);
        eb.aux = w.A;
        eb.lda = sd;
        eb.alpha = coef[2];
        eb.beta = coef[1];
        if (e == cudaSuccess) e = gemm(c, sd, sd, sd, w.A, false, w.A, true, eb, 1);
        // X <- a X + Bm X (wide) or a X + X Bm (tall; Bm is symmetric)
        tc::GemmEp ex = ep_of(tc::GEP_AXPBY, 0, nxt, cols);
        ex.aux = cur;
        ex.lda = cols;
        ex.alpha = 1.0f;
        ex.beta = coef[0];
        if (e == cudaSuccess)
            e = wide ? gemm(c, rows, cols, rows, w.Bm, false, cur, true, ex, 1)
                     : gemm(c, rows, cols, cols, cur, false, w.Bm, true, ex, 1);
        __nv_bfloat16 *t = cur;
        cur = nxt;
        nxt = t;
    }
    return e;
}

cudaError_t tc_effective_rank(int64_t rows, int64_t cols, const void *W, double *out, void *ws, const Ctx &c)
{
    if (!al16(W) || !al16(ws) || encode_fn() == nullptr) return cudaErrorNotSupported;
    const MatrixWs w = matrix_ws(RESBM_OP_EFFECTIVE_RANK, rows, cols, c.sm_count, ws);
    const bool tall = rows >= cols;
    const int64_t sd = tall ? cols : rows, ld = tall ? rows : cols;
    if (sd > tc::kPowMaxN) return cudaErrorNotSupported;
    // the Gram matrix of the smaller side: W^T W (tall) or W W^T (wide), fp32 sums of bf16 products
    tc::ReduceJob job;
    cudaError_t e = tall ? wgrad(c, sd, sd, ld, W, W, w.gram, w.slots, &job)
                         : wgrad(c, sd, sd, ld, W, W, w.gram, w.slots, &job, nullptr, false, false);
    if (e == cudaSuccess) e = reduce_jobs(job, tc::ReduceJob{nullptr, 0, 0, 0, nullptr, 0, 0, 0}, c);
    if (e == cudaSuccess) {
        e = launch(tc::k_power_iter, 1, 1024, 0, c.stream, (const float *)w.gram, (int)sd, 20000, 1e-5f, out);
        count_launches(1);
    }
    return e;
}

namespace tc {
// One thread waits on an mbarrier that nothing arrives on; mbar_wait gives up after kWaitNs,
// sets the timeout bit of the error word and returns, and the kernel exits normally.
__global__ void k_wait_selftest()
{
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&bar), 1);
        fence_mbar_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) mbar_wait(smem_u32(&bar), 0);
}
}  // namespace tc

namespace {
// The 3-D view of the 3-D load form: {64 columns, rows, 64 column blocks} with the blocks 128
// bytes apart, so that one box {64, 128, 2} holds two neighbouring 64-column blocks of 128 rows
// and lands as two 64 x 128 swizzled boxes.
bool make_map_form3d(CUtensorMap *m, const void *ptr, uint64_t rows)
{
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[3] = {64, rows, (cuuint64_t)tc::kFormBlocks};
    cuuint64_t strides[2] = {(cuuint64_t)tc::kFormBlocks * 128, 128};
    cuuint32_t box[3] = {64, 128, 2};
    cuuint32_t es[3] = {1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(ptr), dims, strides, box, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int FORM>
cudaError_t launch_form_load(const CUtensorMap &m, const void *a, int64_t boxes, const Ctx &c)
{
    static std::atomic<uint8_t> smem_set[kMaxDev];
    cudaError_t e = ensure_smem(tc::k_form_load<FORM>, tc::kFormSmem, c.device, smem_set);
    if (e != cudaSuccess) return e;
    tc::k_form_load<FORM><<<c.sm_count, 128, tc::kFormSmem, c.stream>>>(m, static_cast<const uint8_t *>(a), boxes);
    return cudaGetLastError();
}

template <int FORM>
cudaError_t launch_form_store(const CUtensorMap &m, void *b, int64_t boxes, const Ctx &c)
{
    static std::atomic<uint8_t> smem_set[kMaxDev];
    cudaError_t e = ensure_smem(tc::k_form_store<FORM>, tc::kFormSmem, c.device, smem_set);
    if (e != cudaSuccess) return e;
    tc::k_form_store<FORM><<<c.sm_count, 128, tc::kFormSmem, c.stream>>>(m, static_cast<uint8_t *>(b), boxes);
    return cudaGetLastError();
}
}  // namespace

cudaError_t tc_hbm_form(int form, const void *a, void *b, int64_t bytes, const Ctx &c)
{
    const int64_t boxes = bytes / tc::kFormBox, rows = bytes / (tc::kFormBlocks * 128), n16 = bytes / 16;
    const int vgrid = c.sm_count * 4;
    CUtensorMap m;
    std::memset(&m, 0, sizeof(m));
    const bool reads = form == RESBM_HBM_READ_TMA_2D || form == RESBM_HBM_READ_TMA_2D_PAIR ||
                       form == RESBM_HBM_READ_TMA_2D_TILES;
    const bool writes = form == RESBM_HBM_WRITE_TMA_2D || form == RESBM_HBM_WRITE_TMA_2D_TILES;
    if ((reads || writes) && !make_map(&m, reads ? a : b, tc::kFormBlocks * 64, (uint64_t)rows,
                                       tc::kFormBlocks * 128, 64, 128, CU_TENSOR_MAP_SWIZZLE_128B))
        return cudaErrorInvalidValue;
    if (form == RESBM_HBM_READ_TMA_3D && !make_map_form3d(&m, a, (uint64_t)rows)) return cudaErrorInvalidValue;
    cudaError_t e = cudaSuccess;
    switch (form) {
    case RESBM_HBM_READ_V4:
        tc::k_form_read_v4<<<vgrid, 512, 0, c.stream>>>(static_cast<const uint4 *>(a), n16, static_cast<unsigned *>(b));
        e = cudaGetLastError();
        break;
    case RESBM_HBM_WRITE_V4:
        tc::k_form_write_v4<<<vgrid, 512, 0, c.stream>>>(static_cast<uint4 *>(b), n16);
        e = cudaGetLastError();
        break;
    case RESBM_HBM_COPY_V4:
        tc::k_form_copy_v4<<<vgrid, 512, 0, c.stream>>>(static_cast<const uint4 *>(a), static_cast<uint4 *>(b), n16);
        e = cudaGetLastError();
        break;
    case RESBM_HBM_READ_TMA_2D: e = launch_form_load<tc::kLoad2d>(m, a, boxes, c); break;
    case RESBM_HBM_READ_TMA_2D_PAIR: e = launch_form_load<tc::kLoad2dPair>(m, a, boxes, c); break;
    case RESBM_HBM_READ_TMA_3D: e = launch_form_load<tc::kLoad3d>(m, a, boxes, c); break;
    case RESBM_HBM_READ_BULK: e = launch_form_load<tc::kLoadBulk>(m, a, boxes, c); break;
    case RESBM_HBM_WRITE_TMA_2D: e = launch_form_store<tc::kStore2d>(m, b, boxes, c); break;
    case RESBM_HBM_WRITE_BULK: e = launch_form_store<tc::kStoreBulk>(m, b, boxes, c); break;
    case RESBM_HBM_READ_TMA_2D_TILES: e = launch_form_load<tc::kLoadTiles>(m, a, boxes, c); break;
    case RESBM_HBM_WRITE_TMA_2D_TILES: e = launch_form_store<tc::kStoreTiles>(m, b, boxes, c); break;
    default: return cudaErrorInvalidValue;
    }
    count_launches(1);
    return e;
}

cudaError_t tc_wait_selftest(const Ctx &c)
{
    tc::k_wait_selftest<<<1, 32, 0, c.stream>>>();
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t tc_device_error(unsigned int *code, bool clear)
{
    cudaError_t e = cudaMemcpyFromSymbol(code, tc::g_resbm_device_error, sizeof(unsigned int));
    if (e == cudaSuccess && clear && *code) {
        const unsigned int zero = 0;
        e = cudaMemcpyToSymbol(tc::g_resbm_device_error, &zero, sizeof(zero));
    }
    return e;
}

}  // namespace resbm
