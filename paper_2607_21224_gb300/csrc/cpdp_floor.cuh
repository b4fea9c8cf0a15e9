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

}  // namespace cpdp
