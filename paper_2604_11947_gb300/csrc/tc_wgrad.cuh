// tc_wgrad.cuh -- per-CTA weight-gradient partials of the backward kernels.
//
// Each CTA owns a token range and produces, for every 128-row chunk of a d x m weight gradient,
// a 128 x m fp32 partial in TMEM. The epilogue writes it to the CTA's own slot (adding to it for
// the CTA's second and later tile groups, in group order); a second kernel sums the slots in
// slot order, so every element is summed in a fixed order (deterministic) and no CTA ever waits
// for another.
#pragma once

#include "tc_common.cuh"

namespace resbm {
namespace tc {

struct WgradArgs {
    float *slots;   // grid x nch x 128 x M
    int nch;
};

// Called by the 128 epilogue threads with the chunk's row `row` (M values read from TMEM).
template <int M>
__device__ __forceinline__ void wgrad_chunk(const WgradArgs &w, const float (&v)[M], int c, int row,
                                            bool first_group)
{
    float4 *st = reinterpret_cast<float4 *>(w.slots + (((int64_t)blockIdx.x * w.nch + c) * 128 + row) * M);
#pragma unroll
    for (int e = 0; e < M / 4; ++e) {
        float4 x = make_float4(v[4 * e], v[4 * e + 1], v[4 * e + 2], v[4 * e + 3]);
        if (!first_group) {
            const float4 o = st[e];
            x.x = o.x + x.x; x.y = o.y + x.y; x.z = o.z + x.z; x.w = o.w + x.w;
        }
        st_global_hint(&st[e], x, l2_evict_last());   // read back by the reduction soon
    }
}

}  // namespace tc
}  // namespace resbm
