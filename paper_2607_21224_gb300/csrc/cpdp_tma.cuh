// The reconcile (eqs. 2, 6-12) with its rows staged through shared memory by
// the bulk-copy engine (TMA, untiled cp.async.bulk), warp-specialised.
//
// This is an alternative to reconcile_vec4_kernel, kept for comparison and
// off by default (cpdp_set_reconcile_staging). It covers the CPDP method with
// momentum SGD, float32 gradients, no state reconciliation, W <= 16 and N a
// multiple of 4, and computes exactly what reconcile_vec4_kernel computes, in
// the same order, so the two give bit-identical results.
//
// Work unit: a tile of kTmaTile consecutive columns. A persistent CTA takes
// tiles blockIdx.x, blockIdx.x + gridDim.x, ... Its shared memory is a ring of
// `stages` slots; a slot holds one tile of every row the reconcile reads:
// W gradient rows, W parameter rows, W momentum rows, theta_ref and v
// (3W + 2 row segments of kTmaTile floats). Three roles, each with its own
// barriers per slot:
//   - load warp: for each tile, waits until its slot is free (`empty`), lane 0
//     announces the bytes to come on `full`, and the 32 lanes issue one bulk
//     copy per row segment between them;
//   - compute warps (kTmaConsumers threads, one column group of 4 each): wait
//     on `full`, run the reconcile on the slot in place (the same arithmetic
//     as reconcile_vec4_kernel), and arrive on `computed`;
//   - store warp: waits on `computed`, its lanes bulk-store the 2W + 2 updated
//     row segments (parameters, momentum, theta_ref, v) from the slot, wait
//     until their stores have read it, and lane 0 hands the slot back
//     (`empty`).
// Each byte still crosses DRAM once each way; the staging adds a pass through
// shared memory and the cost of issuing one bulk copy per 2 KB row segment.
//
// Every wait is bounded: a wait that has not ended after kTmaWaitLimitNs
// counts itself in tma_wait_timeouts and its warp stops taking tiles, so the
// other roles' waits run out in turn. `withheld_tile` (-1 in normal use) names
// a tile whose loads the load warp leaves out, so that tests can watch these
// limits end the launch. Before returning, the load warp waits
// (again bounded) for every load it issued and the store lanes for all their
// stores, so no copy is in flight into or out of shared memory when the CTA
// exits.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "cpdp_kernels.cuh"

namespace cpdp {

constexpr int kTmaTile = 512;                     // columns (floats) per row segment: 2 KB
constexpr int kTmaConsumers = kTmaTile / 4;       // one float4 column group per compute thread
constexpr int kTmaThreads = kTmaConsumers + 64;   // plus the load warp and the store warp
constexpr int kTmaMaxWorkers = 16;
constexpr unsigned long long kTmaWaitLimitNs = 2000000000ull;  // 2 s

__device__ unsigned long long tma_wait_timeouts;

__device__ __forceinline__ unsigned long long global_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
                 : "memory");
}

// Wait until the phase with parity `parity` of `bar` has completed, for at
// most kTmaWaitLimitNs; false if the limit ran out (counted).
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
    const uint32_t a = smem_addr(bar);
    const unsigned long long start = global_ns();
    while (true) {
        uint32_t done;
        asm volatile(
            "{\n\t.reg .pred p;\n\t"
            "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
            "selp.u32 %0, 1, 0, p;\n\t}"
            : "=r"(done)
            : "r"(a), "r"(parity)
            : "memory");
        if (done) return true;
        if (global_ns() - start > kTmaWaitLimitNs) {
            atomicAdd(&tma_wait_timeouts, 1ull);
            return false;
        }
    }
}

// One bulk copy global -> shared, completing `bytes` on `bar`.
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            smem_addr(dst)),
        "l"(src), "r"(bytes), "r"(smem_addr(bar))
        : "memory");
}

// One bulk copy shared -> global in the current bulk group.
__device__ __forceinline__ void bulk_store(void* dst, const void* src, uint32_t bytes) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst), "r"(smem_addr(src)),
                 "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }

// All but the newest `n` committed store groups have finished reading shared memory.
template <int n>
__device__ __forceinline__ void bulk_wait_read() {
    asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(n) : "memory");
}

// All committed store groups have completed.
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// Make this thread's generic-proxy writes to shared memory visible to the
// bulk-copy (async) proxy.
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Global row segment r of the reconcile's rows: gradients 0..W-1, parameters
// W..2W-1, momentum 2W..3W-1, theta_ref 3W, v 3W+1; `col` is the segment's
// first column, `cols` its length.
__device__ __forceinline__ float* tma_row(float* params, float* mom, const float* grads, float* anchor,
                                          float* slow_v, int W, int64_t N, int r, int64_t col, int cols) {
    // a segment of `cols` elements starting at `off` stays inside a buffer of
    // `extent` elements iff 0 <= off <= extent - cols
    if (r < W) return const_cast<float*>(grads) + CPDP_IDX((int64_t)r * N + col, (int64_t)W * N - cols + 1);
    if (r < 2 * W) return params + CPDP_IDX((int64_t)(r - W) * N + col, (int64_t)W * N - cols + 1);
    if (r < 3 * W) return mom + CPDP_IDX((int64_t)(r - 2 * W) * N + col, (int64_t)W * N - cols + 1);
    return (r == 3 * W ? anchor : slow_v) + CPDP_IDX(col, N - cols + 1);
}

__global__ void __launch_bounds__(kTmaThreads, 1)
reconcile_tma_kernel(float* __restrict__ params, float* __restrict__ mom, const float* __restrict__ grads,
                     float* __restrict__ anchor, float* __restrict__ slow_v, int W, int64_t N, int stages,
                     int64_t withheld_tile, SyncArgs a) {
    extern __shared__ __align__(128) unsigned char tma_smem[];
    const int rows = 3 * W + 2;
    float* slots = reinterpret_cast<float*>(tma_smem);
    uint64_t* full = reinterpret_cast<uint64_t*>(tma_smem + (size_t)stages * rows * kTmaTile * sizeof(float));
    uint64_t* computed = full + stages;
    uint64_t* empty = computed + stages;
    const int64_t ntiles = (N + kTmaTile - 1) / kTmaTile;
    constexpr int kLoadWarp = kTmaConsumers / 32, kStoreWarp = kLoadWarp + 1;

    if (threadIdx.x == 0) {
        for (int s = 0; s < stages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&computed[s], kTmaConsumers);
            mbar_init(&empty[s], 1);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();
    pdl_wait_then_release();

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    if (warp == kLoadWarp) {
        int issued = 0;  // tiles whose loads this CTA issued
        for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x, ++issued) {
            const int s = issued % stages, use = issued / stages;
            bool ok = true;
            if (use > 0 && lane == 0) ok = mbar_wait(&empty[s], (use - 1) & 1);
            if (!__shfl_sync(0xffffffffu, ok, 0)) break;
            const int64_t col = tile * kTmaTile;
            const int cols = (int)(N - col < kTmaTile ? N - col : kTmaTile);
            const uint32_t bytes = (uint32_t)cols * sizeof(float);
            if (tile == withheld_tile) continue;  // a test of the bounded waits: this tile's loads never come
            if (lane == 0) mbar_arrive_expect_tx(&full[s], bytes * rows);
            __syncwarp();
            float* slot = slots + (size_t)s * rows * kTmaTile;
            for (int r = lane; r < rows; r += 32)
                bulk_load(slot + (size_t)r * kTmaTile, tma_row(params, mom, grads, anchor, slow_v, W, N, r, col, cols),
                          bytes, &full[s]);
        }
        // wait for the last load issued into each slot (slots already
        // consumed return at once), so none is in flight when the CTA exits
        if (lane == 0)
            for (int s = 0; s < stages && s < issued; ++s) {
                const int last = s + ((issued - 1 - s) / stages) * stages;
                mbar_wait(&full[s], (last / stages) & 1);
            }
        return;
    }

    if (warp == kStoreWarp) {
        int done = 0;
        for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x, ++done) {
            const int s = done % stages, use = done / stages;
            bool ok = true;
            if (lane == 0) ok = mbar_wait(&computed[s], use & 1);
            if (!__shfl_sync(0xffffffffu, ok, 0)) break;
            const int64_t col = tile * kTmaTile;
            const int cols = (int)(N - col < kTmaTile ? N - col : kTmaTile);
            const uint32_t bytes = (uint32_t)cols * sizeof(float);
            const float* slot = slots + (size_t)s * rows * kTmaTile;
            for (int r = W + lane; r < rows; r += 32)
                bulk_store(tma_row(params, mom, grads, anchor, slow_v, W, N, r, col, cols), slot + (size_t)r * kTmaTile,
                           bytes);
            bulk_commit();
            bulk_wait_read<0>();  // this lane's stores have read the slot
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[s]);
        }
        bulk_wait_all();
        return;
    }

    // compute warps: thread t owns columns 4t..4t+3 of the tile
    const int t = threadIdx.x;
    int done = 0;
    for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x, ++done) {
        const int s = done % stages, use = done / stages;
        if (!mbar_wait(&full[s], use & 1)) break;
        const int64_t col = tile * kTmaTile;
        const int cols = (int)(N - col < kTmaTile ? N - col : kTmaTile);
        float4* slot = reinterpret_cast<float4*>(slots + (size_t)s * rows * kTmaTile);
        constexpr int rq = kTmaTile / 4;  // float4 per row segment
        if (4 * t < cols) {
            float4 gsum = make_float4(0.f, 0.f, 0.f, 0.f);
            for (int i = 0; i < W; ++i) add4(gsum, slot[i * rq + t]);
            const float4 gbar = div4(gsum, a.workers);
            float4 tsum = make_float4(0.f, 0.f, 0.f, 0.f);
            for (int i = 0; i < W; ++i) {
                float4 th = slot[(W + i) * rq + t], bu = slot[(2 * W + i) * rq + t], sv;
                opt_step4<kOptSGD>(gbar, th, bu, sv, a.step);
                slot[(2 * W + i) * rq + t] = bu;
                add4(tsum, th);
            }
            const float4 avg = div4(tsum, a.workers);
            const float4 ref = slot[3 * W * rq + t], vel = slot[(3 * W + 1) * rq + t];
            float4 vn, tn;
            vn.x = fmaf(a.beta, vel.x, avg.x - ref.x);
            vn.y = fmaf(a.beta, vel.y, avg.y - ref.y);
            vn.z = fmaf(a.beta, vel.z, avg.z - ref.z);
            vn.w = fmaf(a.beta, vel.w, avg.w - ref.w);
            tn.x = fmaf(a.alpha, vn.x, ref.x);
            tn.y = fmaf(a.alpha, vn.y, ref.y);
            tn.z = fmaf(a.alpha, vn.z, ref.z);
            tn.w = fmaf(a.alpha, vn.w, ref.w);
            slot[3 * W * rq + t] = tn;
            slot[(3 * W + 1) * rq + t] = vn;
            for (int i = 0; i < W; ++i) slot[(W + i) * rq + t] = tn;
        }
        fence_proxy_async_smem();  // the stores (async proxy) read what this thread wrote
        mbar_arrive(&computed[s]);
    }
}

}  // namespace cpdp
