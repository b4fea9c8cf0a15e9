// The reconcile (eqs. 2, 6-12) with the W worker rows split across the lanes
// of a warp and the W-way sums (eqs. 2 and 7) finished with warp shuffles.
//
// This is an alternative to reconcile_vec4_kernel, kept for comparison and
// off by default (cpdp_set_reconcile_shuffle). It covers the CPDP method with
// momentum SGD, float32 gradients and no state reconciliation, for any W and N
// a multiple of 4.
//
// Mapping: a warp owns a tile of 8 column groups (8 float4, 128 contiguous
// bytes of every row). Lane l takes column group l % 8 and the rows
// l / 8, l / 8 + 4, l / 8 + 8, ...; so one load instruction of the warp reads
// 128 bytes from each of 4 rows. Each lane sums its rows in order; the 4
// partial sums of a column group are then added with two xor shuffles (lanes
// 8 and 16 apart). In that butterfly both partners of a step add the same two
// values, so every lane ends with the same bits and the replicas stay
// bit-identical. From W = 4 on, the order of the W-way sums differs from the
// other kernels' (sequential over the workers), so results agree with them to
// rounding, not bit for bit (up to 3 workers the order is the same). The lane of rows 0, 4, 8, ... (l / 8 == 0) of each column
// group loads theta_ref and v, forms the SlowMo update and passes theta_new to
// the other three lanes of its column group with a shuffle.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "cpdp_kernels.cuh"

namespace cpdp {

constexpr int kShuffleCols = 8;                   // column groups (float4) per warp tile
constexpr int kShuffleRowLanes = 32 / kShuffleCols;  // lanes sharing a column group

__device__ __forceinline__ float4 shfl_xor4(const float4& v, int mask) {
    return make_float4(__shfl_xor_sync(0xffffffffu, v.x, mask), __shfl_xor_sync(0xffffffffu, v.y, mask),
                       __shfl_xor_sync(0xffffffffu, v.z, mask), __shfl_xor_sync(0xffffffffu, v.w, mask));
}

// Sum of the partial sums of the kShuffleRowLanes lanes that share a column group.
__device__ __forceinline__ float4 column_sum(float4 v) {
#pragma unroll
    for (int mask = kShuffleCols; mask < 32; mask <<= 1) add4(v, shfl_xor4(v, mask));
    return v;
}

__global__ void __launch_bounds__(kThreads)
reconcile_shuffle_kernel(float* __restrict__ params, float* __restrict__ mom, const float* __restrict__ grads,
                         float* __restrict__ anchor, float* __restrict__ slow_v, int W, int64_t nq, SyncArgs a) {
    pdl_wait_then_release();
    float4* p4 = reinterpret_cast<float4*>(params);
    float4* m4 = reinterpret_cast<float4*>(mom);
    float4* ref4 = reinterpret_cast<float4*>(anchor);
    float4* vel4 = reinterpret_cast<float4*>(slow_v);
    const int lane = threadIdx.x % 32;
    const int col = lane % kShuffleCols, row0 = lane / kShuffleCols;
    const int64_t warps = (int64_t)gridDim.x * (blockDim.x / 32);
    const int64_t tiles = (nq + kShuffleCols - 1) / kShuffleCols;
    for (int64_t tile = (int64_t)blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32; tile < tiles; tile += warps) {
        const int64_t c = tile * kShuffleCols + col;
        const bool active = c < nq;  // the last tile may be partial; every lane still takes part in the shuffles
        const float4 zero = make_float4(0.f, 0.f, 0.f, 0.f);

        // 1. gradient mean (eq. 2)
        float4 gpart = zero;
        if (active)
            for (int r = row0; r < W; r += kShuffleRowLanes)
                add4(gpart, __ldg(reinterpret_cast<const float4*>(grads) + CPDP_IDX((int64_t)r * nq + c, (int64_t)W * nq)));
        const float4 gbar = div4(column_sum(gpart), a.workers);

        // 2-3. each worker's step with the mean gradient, then the mean of the stepped replicas (eq. 7)
        float4 tpart = zero;
        if (active)
            for (int r = row0; r < W; r += kShuffleRowLanes) {
                const int64_t e = CPDP_IDX((int64_t)r * nq + c, (int64_t)W * nq);
                float4 th = p4[e], bu = m4[e], sv;
                opt_step4<kOptSGD>(gbar, th, bu, sv, a.step);
                m4[e] = bu;
                add4(tpart, th);
            }
        const float4 avg = div4(column_sum(tpart), a.workers);

        // 4. SlowMo (eqs. 8-10), by the lane of rows 0, 4, ... of each column
        // group (lane `col`), which then hands theta_new to the other three
        float4 ref = zero, vel = zero;
        if (active && row0 == 0) {
            ref = ref4[CPDP_IDX(c, nq)];
            vel = vel4[CPDP_IDX(c, nq)];
        }
        float4 vn, tn;
        vn.x = fmaf(a.beta, vel.x, avg.x - ref.x);
        vn.y = fmaf(a.beta, vel.y, avg.y - ref.y);
        vn.z = fmaf(a.beta, vel.z, avg.z - ref.z);
        vn.w = fmaf(a.beta, vel.w, avg.w - ref.w);
        tn.x = fmaf(a.alpha, vn.x, ref.x);
        tn.y = fmaf(a.alpha, vn.y, ref.y);
        tn.z = fmaf(a.alpha, vn.z, ref.z);
        tn.w = fmaf(a.alpha, vn.w, ref.w);
        tn = make_float4(__shfl_sync(0xffffffffu, tn.x, col), __shfl_sync(0xffffffffu, tn.y, col),
                         __shfl_sync(0xffffffffu, tn.z, col), __shfl_sync(0xffffffffu, tn.w, col));
        if (!active) continue;
        if (row0 == 0) {
            ref4[CPDP_IDX(c, nq)] = tn;
            vel4[CPDP_IDX(c, nq)] = vn;
        }

        // 5. write-back to every replica (eqs. 11-12)
        for (int r = row0; r < W; r += kShuffleRowLanes) p4[CPDP_IDX((int64_t)r * nq + c, (int64_t)W * nq)] = tn;
    }
}

}  // namespace cpdp
