// Measurement aids: the floors a launch of the hot path is compared with at
// sizes where launch latency and ramp-up, not bandwidth, decide its time.
//
// floor_stream_kernel is a plain streaming kernel with no optimizer
// arithmetic: per group of 4 columns it reads 4 bf16 values from each of
// n_in_bf16 rows and one float4 from each of n_in float32 rows, adds them,
// and writes the sum to each of n_out rows. Given the same rows as a launch of
// the hot path (in place: the output rows are among the input rows; the
// gradient rows as bf16 rows where the gradients are bf16), it moves the same
// bytes with the same read:write mix over the same buffers; given a
// reconcile's rows, it also walks them column by column as the reconcile does.
// floor_empty_kernel does nothing: it is the cost of a launch.
// Both take part in programmatic dependent launch like the hot-path kernels.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "cpdp_kernels.cuh"

namespace cpdp {

constexpr int kFloorMaxRows = 128;

struct FloorRows {
    const float* in[kFloorMaxRows];
    const bf16_bits* in_bf16[kFloorMaxRows];
    float* out[kFloorMaxRows];
    int n_in, n_in_bf16, n_out;
};

__global__ void __launch_bounds__(kThreads)
floor_stream_kernel(FloorRows rows, int64_t nq) {
    pdl_wait_then_release();
    for (int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; c < nq; c += (int64_t)gridDim.x * blockDim.x) {
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 8
        for (int k = 0; k < rows.n_in_bf16; ++k) add4(acc, GradLoad<bf16_bits>::vec4(rows.in_bf16[k], CPDP_IDX(c, nq)));
#pragma unroll 8
        for (int k = 0; k < rows.n_in; ++k) add4(acc, reinterpret_cast<const float4*>(rows.in[k])[CPDP_IDX(c, nq)]);
#pragma unroll 8
        for (int k = 0; k < rows.n_out; ++k) reinterpret_cast<float4*>(rows.out[k])[CPDP_IDX(c, nq)] = acc;
    }
}

__global__ void __launch_bounds__(kThreads) floor_empty_kernel() { pdl_wait_then_release(); }

// floor_columns_kernel walks a reconcile's rows the way the reconcile does: a
// thread owns a group of 4 columns and visits rows 0 .. W-1 in chunks of CH
// rows, all loads of a chunk in flight together, then theta_ref and v. Each
// row is read and written back in place (the state plus the gradient, so no
// load can be dropped), with no sum over the rows and no dependency between
// them. It moves a CPDP reconcile's bytes in the reconcile's order without its
// arithmetic or its one dependency (the gradient mean before the state rows).
// sq may be null (two state arrays).
template <typename G, int CH, int MIN_BLOCKS>
__global__ void __launch_bounds__(kThreads, MIN_BLOCKS)
floor_columns_kernel(float* __restrict__ params, float* __restrict__ mom, float* __restrict__ sq,
                     const G* __restrict__ grads, float* __restrict__ anchor, float* __restrict__ slow_v, int W,
                     int64_t nq) {
    pdl_wait_then_release();
    float4* p4 = reinterpret_cast<float4*>(params);
    float4* m4 = reinterpret_cast<float4*>(mom);
    float4* s4 = reinterpret_cast<float4*>(sq);
    float4* ref4 = reinterpret_cast<float4*>(anchor);
    float4* vel4 = reinterpret_cast<float4*>(slow_v);
    for (int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; c < nq; c += (int64_t)gridDim.x * blockDim.x) {
        for (int i0 = 0; i0 < W; i0 += CH) {
            float4 th[CH], bu[CH], sv[CH], gr[CH];
#pragma unroll
            for (int k = 0; k < CH; ++k) {
                if (i0 + k < W) {
                    const int64_t e = CPDP_IDX((int64_t)(i0 + k) * nq + c, (int64_t)W * nq);
                    th[k] = p4[e];
                    bu[k] = m4[e];
                    if (s4 != nullptr) sv[k] = s4[e];
                    gr[k] = GradLoad<G>::vec4(grads, e);
                }
            }
#pragma unroll
            for (int k = 0; k < CH; ++k) {
                if (i0 + k < W) {
                    const int64_t e = CPDP_IDX((int64_t)(i0 + k) * nq + c, (int64_t)W * nq);
                    add4(th[k], gr[k]);
                    add4(bu[k], gr[k]);
                    p4[e] = th[k];
                    m4[e] = bu[k];
                    if (s4 != nullptr) {
                        add4(sv[k], gr[k]);
                        s4[e] = sv[k];
                    }
                }
            }
        }
        float4 ref = ref4[CPDP_IDX(c, nq)], vel = vel4[CPDP_IDX(c, nq)];
        add4(ref, vel);
        ref4[CPDP_IDX(c, nq)] = ref;
        vel4[CPDP_IDX(c, nq)] = vel;
    }
}

}  // namespace cpdp
