// tc_wgrad.cuh -- weight-gradient partials of the backward kernels.
//
// Each CTA owns a token range and produces, for every 128-row chunk of a d x m weight gradient,
// a 128 x m fp32 partial in TMEM. The CTAs of a thread-block cluster (1, 2 or 4 CTAs with
// adjacent token ranges) add their partials of a chunk together through distributed shared
// memory: rank k owns rows [k * 128 / cl, (k + 1) * 128 / cl) of the chunk, the other ranks push
// those rows into its receive buffer (st.async, counted on its rx_full barrier), and it adds the
// cl contributions in rank order and writes the sum to the cluster's fp32 slot (adding to it for
// the second and later tile groups, in group order). A second kernel sums the slots in slot
// order. Every element is therefore summed in a fixed order (bitwise reproducible), and the slot
// traffic in HBM is 1 / cl of one slot per CTA.
//
// Exchange protocol, per chunk n (one exchange per chunk and tile group, the same sequence in
// every CTA of the cluster):
//   sender warp (rows owned by rank o != k): wait rx_free[o] of its own CTA (rank o has read
//     exchange n - 1), then st.async its rows into rank o's receive buffer;
//   owner warp: wait rx_full (all bytes of exchange n arrived), read the peers' rows, add in
//     rank order; the owner of local row 0 arms rx_full for exchange n + 1 (arrive.expect_tx),
//     then lane 0 of each owner warp arrives on rx_free[k] of every other rank.
// Both waits are plain CTA-scope mbarrier waits: the data travel by st.async, whose completion
// on the receiver's own barrier makes them visible there, and rx_free only hands a buffer back
// after the values read from it have been consumed. (Cluster-scope release / acquire on these
// arrivals and waits cost more than the halved slot traffic saves.)
// The kernels send a chunk as soon as its accumulator is complete but receive it part of a chunk
// later (the owner rows stay in a third TMEM accumulator meanwhile), so the exchange's latency
// and the CTAs' skew are off the critical path. rx_full is armed for exchange 0 before a
// cluster-wide barrier at kernel start, and the kernel ends with a cluster-wide barrier, so no
// CTA touches a peer's shared memory before it is set up or after it has left. Every wait is
// bounded.
#pragma once

#include "tc_common.cuh"

namespace resbm {
namespace tc {

struct WgradArgs {
    float *slots;   // clusters x nch x 128 x M
    int nch;
};

// Receive buffer for up to four CTAs per cluster: (cl - 1) x (128 / cl) rows of M fp32, at most
// 96 rows (cl = 4; 64 for cl = 2).
template <int M> constexpr uint32_t wgrad_rx_bytes(int clmax)
{
    return clmax <= 1 ? 0u : (uint32_t)((clmax - 1) * (128 / clmax) * M * 4);
}

// CLMAX: the largest cluster the kernel is built for (1: the exchange is compiled out).
template <int M, int CLMAX> struct WgradXchg {
    static constexpr int V4 = M / 4;   // float4 per row
    uint32_t cl, rank, cid;            // CTAs per cluster, this CTA's rank, cluster index
    uint32_t rx;                       // receive buffer (shared address)
    uint32_t rx_full;                  // barrier: bytes of the current exchange received
    uint32_t rx_free;                  // barriers rx_free[0 .. 3]: rank o has read my rows
    uint32_t n;                        // exchanges so far

    __device__ __forceinline__ uint32_t rx_bytes() const { return (cl - 1) * (128 / cl) * M * 4; }

    // Initialization by one thread, after mbar_init of the kernel's own barriers and before the
    // fence_mbar_init and the cluster-wide barrier: rx_full takes one arrival (its arming) plus
    // the exchange's bytes, rx_free[o] the (128 / cl) / 32 owner warps of rank o.
    __device__ __forceinline__ void init_barriers() const
    {
        if (CLMAX <= 1 || cl <= 1) return;
        mbar_init(rx_full, 1);
        for (int o = 0; o < 4; ++o) mbar_init(rx_free + 8 * o, (128 / cl) / 32);
    }
    // Arms rx_full for exchange 0 (the thread that initialized it, after fence_mbar_init).
    __device__ __forceinline__ void arm_first() const
    {
        if (CLMAX > 1 && cl > 1) mbar_expect_tx(rx_full, rx_bytes());
    }

    // Whether this launch exchanges partials (clusters of more than one CTA), and whether the
    // thread whose TMEM lane is chunk row `row` owns that row (adds the cluster's contributions
    // and writes the slot) or sends it to the owning CTA. Owner rows are whole warps.
    __device__ __forceinline__ bool exchanging() const { return CLMAX > 1 && cl > 1; }
    __device__ __forceinline__ bool owns(int row) const
    {
        return !exchanging() || (uint32_t)(row / (128 / (int)cl)) == rank;
    }

    // Sender: push chunk row `row` (partial v) into the owner's receive buffer. False if the
    // wait for the owner's previous exchange gave up.
    __device__ __forceinline__ bool send(const float (&v)[M], int row)
    {
        const uint32_t ph = n & 1;
        ++n;
        const int rs = 128 / (int)cl;
        const uint32_t o = (uint32_t)(row / rs);
        const int lr = row - (int)o * rs;
        if (!mbar_wait(rx_free + 8 * o, ph ^ 1)) return false;
        const uint32_t ps = rank < o ? rank : rank - 1;
        const uint32_t dst = map_shared(rx + (ps * rs + lr) * (uint32_t)(M * 4), o);
        const uint32_t bar = map_shared(rx_full, o);
#pragma unroll
        for (int e = 0; e < V4; ++e)
            st_async_f4(dst + 16u * (uint32_t)(e ^ (lr & (V4 - 1))),
                        make_float4(v[4 * e], v[4 * e + 1], v[4 * e + 2], v[4 * e + 3]), bar);
        return true;
    }

    // Owner: wait for the peers' rows of the exchange, add the cl contributions in rank order
    // (v is this CTA's), re-arm rx_full, hand the receive buffer back to the senders and write
    // the sum to chunk c of the cluster's slot. Called by whole warps; false if the wait gave up.
    __device__ __forceinline__ bool receive(const WgradArgs &w, const float (&v)[M], int c, int row, bool first_group)
    {
        const uint32_t ph = n & 1;
        ++n;
        const int rs = 128 / (int)cl;
        const int lr = row - (int)rank * rs;
        // (warp-uniform outcome: the warp synchronizes below)
        if (!__all_sync(0xffffffffu, mbar_wait(rx_full, ph))) return false;
        float4 s[V4];
        for (uint32_t p = 0; p < cl; ++p) {
            float4 x[V4];
            if (p == rank) {
#pragma unroll
                for (int e = 0; e < V4; ++e) x[e] = make_float4(v[4 * e], v[4 * e + 1], v[4 * e + 2], v[4 * e + 3]);
            } else {
                const uint32_t src = rx + ((p < rank ? p : p - 1) * rs + lr) * (uint32_t)(M * 4);
#pragma unroll
                for (int e = 0; e < V4; ++e) {
                    asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
                                 : "=f"(x[e].x), "=f"(x[e].y), "=f"(x[e].z), "=f"(x[e].w)
                                 : "r"(src + 16u * (uint32_t)(e ^ (lr & (V4 - 1))))
                                 : "memory");
                }
            }
#pragma unroll
            for (int e = 0; e < V4; ++e) {
                if (p == 0) {
                    s[e] = x[e];
                } else {
                    s[e].x = s[e].x + x[e].x; s[e].y = s[e].y + x[e].y;
                    s[e].z = s[e].z + x[e].z; s[e].w = s[e].w + x[e].w;
                }
            }
        }
        if (lr == 0) mbar_expect_tx(rx_full, rx_bytes());   // arm the next exchange
        __syncwarp();
        if ((row & 31) == 0)
            for (uint32_t p = 0; p < cl; ++p)
                if (p != rank) mbar_arrive_remote(map_shared(rx_free + 8 * rank, p));
        store(w, s, c, row, first_group);
        return true;
    }

    // Without an exchange: chunk row `row` straight into the CTA's slot.
    __device__ __forceinline__ void store_own(const WgradArgs &w, const float (&v)[M], int c, int row, bool first_group) const
    {
        float4 s[V4];
#pragma unroll
        for (int e = 0; e < V4; ++e) s[e] = make_float4(v[4 * e], v[4 * e + 1], v[4 * e + 2], v[4 * e + 3]);
        store(w, s, c, row, first_group);
    }

    __device__ __forceinline__ void store(const WgradArgs &w, float4 (&s)[V4], int c, int row, bool first_group) const
    {
        float4 *st = reinterpret_cast<float4 *>(w.slots + (((int64_t)cid * w.nch + c) * 128 + row) * M);
#pragma unroll
        for (int e = 0; e < V4; ++e) {
            float4 x = s[e];
            if (!first_group) {
                const float4 o = st[e];
                x.x = o.x + x.x; x.y = o.y + x.y; x.z = o.z + x.z; x.w = o.w + x.w;
            }
            st_global_hint(&st[e], x, l2_evict_last());   // read back by the reduction soon
        }
    }
};

}  // namespace tc
}  // namespace resbm
