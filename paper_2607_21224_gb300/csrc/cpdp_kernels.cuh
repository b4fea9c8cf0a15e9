// Device kernels of libcpdp: the data-parallel hot path of CPDP on one GB300.
//
// W workers' replicas are rows of [W][N] float32 buffers in HBM. Every kernel
// here is elementwise in the parameter index j, with a reduction only over the
// W rows of one column, so each kernel streams its bytes once: it is bound by
// HBM bandwidth, not by arithmetic (about 0.3 flop per byte). No tensor cores:
// nothing here is a dense contraction.
//
// Access pattern: one thread owns a group of 4 consecutive parameters (one
// 128-bit vector per row). A warp therefore reads or writes 512 contiguous
// bytes of each row it touches; the W-way "strided" reads of the reconcile are
// W such coalesced segments, one per row, and the W-way sums stay in the
// thread's registers (no shared memory, no shuffles). Gradients are read
// through the read-only path; state is read and written with plain
// write-back accesses. Evict-first (streaming) hints measured slower here: the
// reconcile lost 6 % with them, because dirty lines pushed out of L2 early
// reach DRAM as scattered writes instead of combining per DRAM page.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace cpdp {

constexpr int kThreads = 256;

// Optimizers each worker can run (the paper: SGD with momentum for ResNet-50,
// AdamW for ViT-S; Sec. 5.2, Table 3).
constexpr int kOptSGD = 0;
constexpr int kOptAdamW = 1;

// Per-step scalars of AdamW, computed on the host in double precision for the
// current step count t and rounded to float:
//   decay = 1 - lr * wd, step_size = lr / (1 - beta1^t), inv_bc2_sqrt = 1 / sqrt(1 - beta2^t).
struct AdamArgs {
    float decay;
    float step_size;
    float inv_bc2_sqrt;
    float beta1, one_minus_beta1;
    float beta2, one_minus_beta2;
    float eps;
};

// Hyperparameters of the optimizer step. SGD (Sec. 4.2, Table 3): PyTorch SGD
// with momentum and coupled weight decay, no dampening, no Nesterov term.
// AdamW: the `adam` scalars above (lr and weight decay enter through them).
struct StepArgs {
    float lr;
    float momentum;
    float weight_decay;
    AdamArgs adam;
};

// Hyperparameters of the reconcile: the step above plus SlowMo (eqs. 8-10)
// and the worker count used by both means (eqs. 2 and 7).
struct SyncArgs {
    StepArgs step;
    float beta;
    float alpha;
    float workers;  // W as float; the means divide by it (one IEEE division)
};

// bfloat16 gradients are stored as raw 16-bit patterns; widening to float32 is
// exact (the bf16 bits are the upper half of the float32 bits).
struct bf16_bits {
    uint16_t bits;
};

__device__ __forceinline__ float bf16_widen(uint16_t b) {
    return __uint_as_float(static_cast<uint32_t>(b) << 16);
}

// Index checks for a debug build (compiled with -DCPDP_CHECKED): every global
// memory index is compared with the extent of the buffer it addresses. One
// outside it is counted in bad_index_count and replaced by 0, so the access
// stays inside the buffer and nothing traps. Without CPDP_CHECKED the index is
// used as it is and the kernels compile as if the macro were absent.
#ifdef CPDP_CHECKED
__device__ unsigned long long bad_index_count;
__device__ __forceinline__ int64_t checked_index(int64_t i, int64_t extent) {
    if (i < 0 || i >= extent) {
        atomicAdd(&bad_index_count, 1ull);
        return 0;
    }
    return i;
}
#define CPDP_IDX(i, extent) ::cpdp::checked_index((i), (extent))
#else
#define CPDP_IDX(i, extent) (i)
#endif

template <typename G>
struct GradLoad;

template <>
struct GradLoad<float> {
    // q indexes groups of 4 elements
    static __device__ __forceinline__ float4 vec4(const float* g, int64_t q) {
        return __ldg(reinterpret_cast<const float4*>(g) + q);
    }
    static __device__ __forceinline__ float one(const float* g, int64_t e) { return __ldg(g + e); }
    // the group's raw words, widened only when summed (identical for float32)
    using Words = float4;
    static __device__ __forceinline__ Words words(const float* g, int64_t q) { return vec4(g, q); }
    static __device__ __forceinline__ float4 widen(const Words& w) { return w; }
};

template <>
struct GradLoad<bf16_bits> {
    static __device__ __forceinline__ float4 vec4(const bf16_bits* g, int64_t q) {
        const uint2 u = __ldg(reinterpret_cast<const uint2*>(g) + q);
        return make_float4(__uint_as_float(u.x << 16), __uint_as_float(u.x & 0xffff0000u),
                           __uint_as_float(u.y << 16), __uint_as_float(u.y & 0xffff0000u));
    }
    static __device__ __forceinline__ float one(const bf16_bits* g, int64_t e) {
        return bf16_widen(__ldg(reinterpret_cast<const unsigned short*>(g) + e));
    }
    // the group's 8 raw bytes (2 registers instead of 4 while a chunk is in flight)
    using Words = uint2;
    static __device__ __forceinline__ Words words(const bf16_bits* g, int64_t q) {
        return __ldg(reinterpret_cast<const uint2*>(g) + q);
    }
    static __device__ __forceinline__ float4 widen(const Words& u) {
        return make_float4(__uint_as_float(u.x << 16), __uint_as_float(u.x & 0xffff0000u),
                           __uint_as_float(u.y << 16), __uint_as_float(u.y & 0xffff0000u));
    }
};

// One element of one worker's optimizer.step():
//   d = g + wd * theta;  buf = mu * buf + d;  theta = theta - lr * buf
// (each line one fused multiply-add, so one rounding per line).
__device__ __forceinline__ void sgd_momentum(float g, float& theta, float& buf, const StepArgs& a) {
    const float d = fmaf(a.weight_decay, theta, g);
    buf = fmaf(a.momentum, buf, d);
    theta = fmaf(-a.lr, buf, theta);
}

__device__ __forceinline__ void add4(float4& acc, const float4& x) {
    acc.x += x.x;
    acc.y += x.y;
    acc.z += x.z;
    acc.w += x.w;
}

__device__ __forceinline__ float4 div4(const float4& x, float w) {
    return make_float4(x.x / w, x.y / w, x.z / w, x.w / w);
}

// One element of one worker's AdamW step (decoupled weight decay, bias-
// corrected moments; m is the first moment, s the second):
//   theta *= decay;  m = b1 m + (1-b1) g;  s = b2 s + (1-b2) g^2;
//   theta -= step_size * m / (sqrt(s) / sqrt(1 - beta2^t) + eps)
// The division by sqrt(1 - beta2^t) is a multiplication by its reciprocal,
// formed on the host, and m / denom uses the fast-division intrinsic (a few
// ulps): with bf16 gradients the step is issue-bound, and the two IEEE
// divisions it replaces cost 2.5 % of its bandwidth.
__device__ __forceinline__ void adamw(float g, float& theta, float& m, float& s, const AdamArgs& a) {
    theta = theta * a.decay;
    m = fmaf(a.beta1, m, a.one_minus_beta1 * g);
    s = fmaf(a.beta2, s, a.one_minus_beta2 * (g * g));
    const float denom = fmaf(sqrtf(s), a.inv_bc2_sqrt, a.eps);
    theta = fmaf(-a.step_size, __fdividef(m, denom), theta);
}

// The worker's optimizer step, chosen at compile time. `s` is unused by SGD.
template <int OPT>
__device__ __forceinline__ void opt_step(float g, float& theta, float& m, float& s, const StepArgs& a) {
    if (OPT == kOptAdamW)
        adamw(g, theta, m, s, a.adam);
    else
        sgd_momentum(g, theta, m, a);
}

template <int OPT>
__device__ __forceinline__ void opt_step4(const float4& g, float4& theta, float4& m, float4& s, const StepArgs& a) {
    opt_step<OPT>(g.x, theta.x, m.x, s.x, a);
    opt_step<OPT>(g.y, theta.y, m.y, s.y, a);
    opt_step<OPT>(g.z, theta.z, m.z, s.z, a);
    opt_step<OPT>(g.w, theta.w, m.w, s.w, a);
}

// Programmatic dependent launch. Every kernel here starts by waiting until
// the grid it follows on the stream has completed and its writes are visible
// (griddepcontrol.wait), and then lets the next launch on the stream begin
// scheduling its blocks (griddepcontrol.launch_dependents). The next grid's
// blocks can then take SMs as this grid's last wave drains, and its launch
// latency is hidden; they still wait for this grid's completion before
// touching memory. Both instructions are no-ops in a launch without the
// programmatic-serialization attribute.
__device__ __forceinline__ void pdl_wait_then_release() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// ---------------------------------------------------------------------------
// K0: Algorithm 1 initialisation. theta_i = theta0 for every worker,
// theta_ref = theta0, v = 0, buf_i = 0 (and the AdamW second moments, when
// `sq` is not null).
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads)
init_vec4_kernel(float* __restrict__ params, float* __restrict__ mom, float* __restrict__ sq,
                 float* __restrict__ anchor, float* __restrict__ slow_v, const float* __restrict__ theta0,
                 int W, int64_t nq) {
    pdl_wait_then_release();
    const float4 zero = make_float4(0.f, 0.f, 0.f, 0.f);
    float4* p4 = reinterpret_cast<float4*>(params);
    float4* m4 = reinterpret_cast<float4*>(mom);
    float4* s4 = reinterpret_cast<float4*>(sq);
    for (int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; c < nq;
         c += (int64_t)gridDim.x * blockDim.x) {
        const float4 t0 = __ldg(reinterpret_cast<const float4*>(theta0) + CPDP_IDX(c, nq));
        for (int i = 0; i < W; ++i) {
            p4[CPDP_IDX((int64_t)i * nq + c, (int64_t)W * nq)] = t0;
            m4[CPDP_IDX((int64_t)i * nq + c, (int64_t)W * nq)] = zero;
            if (s4 != nullptr) s4[CPDP_IDX((int64_t)i * nq + c, (int64_t)W * nq)] = zero;
        }
        reinterpret_cast<float4*>(anchor)[CPDP_IDX(c, nq)] = t0;
        reinterpret_cast<float4*>(slow_v)[CPDP_IDX(c, nq)] = zero;
    }
}

__global__ void __launch_bounds__(kThreads)
init_scalar_kernel(float* __restrict__ params, float* __restrict__ mom, float* __restrict__ sq,
                   float* __restrict__ anchor, float* __restrict__ slow_v, const float* __restrict__ theta0,
                   int W, int64_t N) {
    pdl_wait_then_release();
    for (int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; j < N;
         j += (int64_t)gridDim.x * blockDim.x) {
        const float t0 = theta0[CPDP_IDX(j, N)];
        for (int i = 0; i < W; ++i) {
            params[CPDP_IDX((int64_t)i * N + j, (int64_t)W * N)] = t0;
            mom[CPDP_IDX((int64_t)i * N + j, (int64_t)W * N)] = 0.f;
            if (sq != nullptr) sq[CPDP_IDX((int64_t)i * N + j, (int64_t)W * N)] = 0.f;
        }
        anchor[CPDP_IDX(j, N)] = t0;
        slow_v[CPDP_IDX(j, N)] = 0.f;
    }
}

// ---------------------------------------------------------------------------
// K1: local update phase (eq. 5 with the worker's optimizer step). Every
// worker's row uses its own gradient row, and the [W][N] arrays share one
// layout, so the step is one flat elementwise pass over W*N elements. Bytes
// per element: SGD 12 read + 8 written with float32 gradients (10 + 8 with
// bf16); AdamW 16 + 12 (14 + 12). U vectors of 4 per thread per iteration, all
// loads issued before any store.
// ---------------------------------------------------------------------------
// AdamW's step is compiled for 4 resident blocks (64 registers): at 3 blocks
// it measured 10 % slower with bf16 gradients, where its extra arithmetic per
// byte makes it latency- rather than bandwidth-limited.
template <int OPT>
struct LocalStepBlocks {
    static constexpr int value = OPT == kOptAdamW ? 4 : 1;
};

// WARP_RUNS picks which U vectors a thread takes: with it, each warp streams
// U * 512 contiguous bytes of every array (vectors 32 apart); without it, the
// block's 256 threads cover 4 KB and a thread's vectors are 4 KB apart.
template <int OPT, typename G, int U, bool WARP_RUNS>
__global__ void __launch_bounds__(kThreads, LocalStepBlocks<OPT>::value)
local_step_kernel(float* __restrict__ params, float* __restrict__ mom, float* __restrict__ sq,
                  const G* __restrict__ grads, int64_t total, StepArgs a) {
    pdl_wait_then_release();
    const int64_t nq = total >> 2;
    float4* p4 = reinterpret_cast<float4*>(params);
    float4* m4 = reinterpret_cast<float4*>(mom);
    float4* s4 = reinterpret_cast<float4*>(sq);
    const int64_t stride = (int64_t)gridDim.x * blockDim.x * U;
    const int64_t first = WARP_RUNS ? (int64_t)(threadIdx.x / 32) * 32 * U + threadIdx.x % 32 : threadIdx.x;
    const int64_t step = WARP_RUNS ? 32 : blockDim.x;
    for (int64_t q0 = (int64_t)blockIdx.x * blockDim.x * U + first; q0 < nq; q0 += stride) {
        float4 th[U], bu[U], sv[U], gr[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int64_t q = q0 + (int64_t)u * step;
            if (q < nq) {
                th[u] = p4[CPDP_IDX(q, nq)];
                bu[u] = m4[CPDP_IDX(q, nq)];
                if (OPT == kOptAdamW) sv[u] = s4[CPDP_IDX(q, nq)];
                gr[u] = GradLoad<G>::vec4(grads, CPDP_IDX(q, nq));
            }
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int64_t q = q0 + (int64_t)u * step;
            if (q < nq) {
                opt_step4<OPT>(gr[u], th[u], bu[u], sv[u], a);
                m4[CPDP_IDX(q, nq)] = bu[u];
                if (OPT == kOptAdamW) s4[CPDP_IDX(q, nq)] = sv[u];
                p4[CPDP_IDX(q, nq)] = th[u];
            }
        }
    }
    // ragged tail: the last total % 4 elements, one thread each in block 0
    if (blockIdx.x == 0) {
        const int64_t e = (nq << 2) + threadIdx.x;
        if (e < total) {
            float th = params[CPDP_IDX(e, total)], bu = mom[CPDP_IDX(e, total)], sv = 0.f;
            if (OPT == kOptAdamW) sv = sq[CPDP_IDX(e, total)];
            opt_step<OPT>(GradLoad<G>::one(grads, CPDP_IDX(e, total)), th, bu, sv, a);
            mom[CPDP_IDX(e, total)] = bu;
            if (OPT == kOptAdamW) sq[CPDP_IDX(e, total)] = sv;
            params[CPDP_IDX(e, total)] = th;
        }
    }
}

// ---------------------------------------------------------------------------
// K2: synchronization step, fused into one pass per column of 4 parameters.
//
// Method kMethodCPDP (eqs. 2, 6-12; Algorithm 1's sync branch):
//   1. gbar = (1/W) sum_i g_i                           reads W gradient rows
//   2. per worker: momentum step with gbar on theta_i   reads theta_i, buf_i,
//      and buf_i; theta'_i kept in registers            writes buf_i
//   3. theta_avg = (1/W) sum_i theta'_i
//   4. v = beta v + (theta_avg - theta_ref); theta_new = theta_ref + alpha v
//   5. theta_i = theta_new for all i, theta_ref = theta_new, v stored
//   12W + 8 bytes read and 8W + 8 written per parameter (float32 gradients).
// Method kMethodLocalSGD (the paper's LocalSGD baseline, Sec. 5.4): step 1 is
//   skipped, step 2 uses each worker's own gradient, steps 3 and 5 write
//   theta_avg to every replica, step 4 is skipped (no anchor, no velocity):
//   12W read and 8W written per parameter.
// Method kMethodDDP (the paper's DDP baseline, K = 1): steps 1-2 only, each
//   worker keeps its own stepped theta'_i (no parameter mean): 12W read and 8W
//   written per parameter.
// With OPT = kOptAdamW the worker's step is AdamW and each row also reads and
// writes its second moments (4W more bytes each way).
// With STATE_SYNC (CPDP and LocalSGD only), the optimizer-state reconciliation
// variant: instead of each worker's own post-step state, the mean over the
// workers of the momentum buffers (and AdamW second moments) is written to
// every worker; the byte count is unchanged.
// Rows are visited in chunks of CH so that a chunk's loads are all in flight
// together while register use stays bounded for any W. LATE_ANCHOR loads
// theta_ref and v after the rows instead of before them: one more dependent
// load at the end, but 8 fewer registers live across the row loops, which lets
// the register-heavy variants run more blocks per SM. Idx is the type of the
// column and row-offset arithmetic: int32_t where W * N / 4 plus the grid's
// thread count stays below 2^31 (the host checks), which frees the registers a
// 64-bit offset takes, else int64_t. GCH is the number of gradient rows per
// load chunk of step 1 (CH by default); where it differs from CH the gradient
// rows are held as raw words until summed, and OVERLAP also issues the first
// state chunk's loads together with the first gradient chunk, so that they
// are in flight while the gradient sum completes. Neither changes the order of
// any sum, so the results are bit-identical for every GCH and OVERLAP. Where
// the replicas are written from one register (CPDP, LocalSGD) the rows are
// bit-identical after the launch.
// ---------------------------------------------------------------------------
constexpr int kMethodCPDP = 0;
constexpr int kMethodLocalSGD = 1;
constexpr int kMethodDDP = 2;

// Steps 2-3 of the reconcile below for the chunk of rows i0 .. i0 + CH - 1 of
// column group c, the rows already in registers: each worker's optimizer step
// (with gbar, or with its own gradient gw for LocalSGD), its state written
// back or added to the state sums, its parameters written back (DDP) or added
// to the parameter sum.
template <int METHOD, int OPT, bool STATE_SYNC, int CH, typename Idx>
__device__ __forceinline__ void reconcile_chunk(int i0, int W, Idx nq, Idx c, float4* p4, float4* m4, float4* s4,
                                                const float4& gbar, const StepArgs& step, float4 (&th)[CH],
                                                float4 (&bu)[CH], float4 (&sv)[CH], const float4 (&gw)[CH],
                                                float4& tsum, float4& bsum, float4& ssum) {
#pragma unroll
    for (int k = 0; k < CH; ++k) {
        if (i0 + k < W) {
            opt_step4<OPT>(METHOD == kMethodLocalSGD ? gw[k] : gbar, th[k], bu[k], sv[k], step);
            if (STATE_SYNC) {
                add4(bsum, bu[k]);
                if (OPT == kOptAdamW) add4(ssum, sv[k]);
            } else {
                m4[CPDP_IDX((Idx)(i0 + k) * nq + c, (Idx)W * nq)] = bu[k];
                if (OPT == kOptAdamW) s4[CPDP_IDX((Idx)(i0 + k) * nq + c, (Idx)W * nq)] = sv[k];
            }
            if (METHOD == kMethodDDP)
                p4[CPDP_IDX((Idx)(i0 + k) * nq + c, (Idx)W * nq)] = th[k];
            else
                add4(tsum, th[k]);
        }
    }
}

template <int METHOD, int OPT, bool STATE_SYNC, typename G, int CH, int MIN_BLOCKS, bool LATE_ANCHOR, typename Idx,
          int GCH = CH, bool OVERLAP = false>
__global__ void __launch_bounds__(kThreads, MIN_BLOCKS)
reconcile_vec4_kernel(float* __restrict__ params, float* __restrict__ mom, float* __restrict__ sq,
                      const G* __restrict__ grads, float* __restrict__ anchor, float* __restrict__ slow_v,
                      int W, Idx nq, SyncArgs a) {
    static_assert(!(STATE_SYNC && METHOD == kMethodDDP), "DDP's states are identical across workers");
    static_assert(!(OVERLAP && METHOD == kMethodLocalSGD), "LocalSGD has no gradient mean to overlap");
    pdl_wait_then_release();
    float4* p4 = reinterpret_cast<float4*>(params);
    float4* m4 = reinterpret_cast<float4*>(mom);
    float4* s4 = reinterpret_cast<float4*>(sq);
    float4* ref4 = reinterpret_cast<float4*>(anchor);
    float4* vel4 = reinterpret_cast<float4*>(slow_v);
    for (Idx c = (Idx)blockIdx.x * blockDim.x + threadIdx.x; c < nq; c += (Idx)gridDim.x * blockDim.x) {
        float4 ref, vel;
        if (METHOD == kMethodCPDP && !LATE_ANCHOR) {
            ref = ref4[CPDP_IDX(c, nq)];
            vel = vel4[CPDP_IDX(c, nq)];
        }

        // 1. gradient mean (eq. 2)
        float4 gbar = make_float4(0.f, 0.f, 0.f, 0.f);
        // the rows of the current state chunk (the first one loaded in step 1 when OVERLAP)
        float4 th[CH], bu[CH], sv[CH];
        if (METHOD != kMethodLocalSGD) {
            float4 gsum = make_float4(0.f, 0.f, 0.f, 0.f);
            if constexpr (GCH == CH && !OVERLAP) {
                for (int i0 = 0; i0 < W; i0 += CH) {
                    float4 gv[CH];
#pragma unroll
                    for (int k = 0; k < CH; ++k)
                        if (i0 + k < W) gv[k] = GradLoad<G>::vec4(grads, CPDP_IDX((Idx)(i0 + k) * nq + c, (Idx)W * nq));
#pragma unroll
                    for (int k = 0; k < CH; ++k)
                        if (i0 + k < W) add4(gsum, gv[k]);
                }
            } else {
                for (int i0 = 0; i0 < W; i0 += GCH) {
                    typename GradLoad<G>::Words gv[GCH];
#pragma unroll
                    for (int k = 0; k < GCH; ++k)
                        if (i0 + k < W) gv[k] = GradLoad<G>::words(grads, CPDP_IDX((Idx)(i0 + k) * nq + c, (Idx)W * nq));
                    if (OVERLAP && i0 == 0) {
#pragma unroll
                        for (int k = 0; k < CH; ++k) {
                            if (k < W) {
                                th[k] = p4[CPDP_IDX((Idx)k * nq + c, (Idx)W * nq)];
                                bu[k] = m4[CPDP_IDX((Idx)k * nq + c, (Idx)W * nq)];
                                if (OPT == kOptAdamW) sv[k] = s4[CPDP_IDX((Idx)k * nq + c, (Idx)W * nq)];
                            }
                        }
                    }
#pragma unroll
                    for (int k = 0; k < GCH; ++k)
                        if (i0 + k < W) add4(gsum, GradLoad<G>::widen(gv[k]));
                }
            }
            gbar = div4(gsum, a.workers);
        }

        // 2-3. optimizer step on every worker (eq. 6: with gbar; LocalSGD: with
        // its own gradient), then the mean of the stepped replicas (eq. 7)
        float4 tsum = make_float4(0.f, 0.f, 0.f, 0.f);
        float4 bsum = make_float4(0.f, 0.f, 0.f, 0.f), ssum = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int i0 = 0; i0 < W; i0 += CH) {
            float4 gw[CH];
            if (!(OVERLAP && i0 == 0)) {
#pragma unroll
                for (int k = 0; k < CH; ++k) {
                    if (i0 + k < W) {
                        th[k] = p4[CPDP_IDX((Idx)(i0 + k) * nq + c, (Idx)W * nq)];
                        bu[k] = m4[CPDP_IDX((Idx)(i0 + k) * nq + c, (Idx)W * nq)];
                        if (OPT == kOptAdamW) sv[k] = s4[CPDP_IDX((Idx)(i0 + k) * nq + c, (Idx)W * nq)];
                        if (METHOD == kMethodLocalSGD) gw[k] = GradLoad<G>::vec4(grads, CPDP_IDX((Idx)(i0 + k) * nq + c, (Idx)W * nq));
                    }
                }
            }
            reconcile_chunk<METHOD, OPT, STATE_SYNC, CH, Idx>(i0, W, nq, c, p4, m4, s4, gbar, a.step, th, bu, sv, gw, tsum,
                                                              bsum, ssum);
        }
        if (METHOD == kMethodDDP) continue;
        if (STATE_SYNC) {
            const float4 bmean = div4(bsum, a.workers);
            for (int i = 0; i < W; ++i) m4[CPDP_IDX((Idx)i * nq + c, (Idx)W * nq)] = bmean;
            if (OPT == kOptAdamW) {
                const float4 smean = div4(ssum, a.workers);
                for (int i = 0; i < W; ++i) s4[CPDP_IDX((Idx)i * nq + c, (Idx)W * nq)] = smean;
            }
        }
        const float4 avg = div4(tsum, a.workers);

        // 4. SlowMo (eqs. 8-10); LocalSGD writes the plain average
        float4 tn = avg;
        if (METHOD == kMethodCPDP) {
            if (LATE_ANCHOR) {
                ref = ref4[CPDP_IDX(c, nq)];
                vel = vel4[CPDP_IDX(c, nq)];
            }
            float4 vn;
            vn.x = fmaf(a.beta, vel.x, avg.x - ref.x);
            vn.y = fmaf(a.beta, vel.y, avg.y - ref.y);
            vn.z = fmaf(a.beta, vel.z, avg.z - ref.z);
            vn.w = fmaf(a.beta, vel.w, avg.w - ref.w);
            tn.x = fmaf(a.alpha, vn.x, ref.x);
            tn.y = fmaf(a.alpha, vn.y, ref.y);
            tn.z = fmaf(a.alpha, vn.z, ref.z);
            tn.w = fmaf(a.alpha, vn.w, ref.w);
            ref4[CPDP_IDX(c, nq)] = tn;
            vel4[CPDP_IDX(c, nq)] = vn;
        }

        // 5. write-back to every replica (eqs. 11-12)
        for (int i = 0; i < W; ++i) p4[CPDP_IDX((Idx)i * nq + c, (Idx)W * nq)] = tn;
    }
}

// The same reconcile for at most WMAX workers, in one round trip to memory:
// every row the column needs (the W gradient rows, the W rows of each state
// array, theta_ref and v) is loaded before any of them is used, where
// reconcile_vec4_kernel finishes the gradient mean before it loads the state
// rows. The sums run over the workers in the same order, so the results are
// bit-identical to reconcile_vec4_kernel's.
template <int METHOD, int OPT, bool STATE_SYNC, typename G, int WMAX, int MIN_BLOCKS>
__global__ void __launch_bounds__(kThreads, MIN_BLOCKS)
reconcile_onepass_kernel(float* __restrict__ params, float* __restrict__ mom, float* __restrict__ sq,
                         const G* __restrict__ grads, float* __restrict__ anchor, float* __restrict__ slow_v,
                         int W, int64_t nq, SyncArgs a) {
    static_assert(!(STATE_SYNC && METHOD == kMethodDDP), "DDP's states are identical across workers");
    pdl_wait_then_release();
    float4* p4 = reinterpret_cast<float4*>(params);
    float4* m4 = reinterpret_cast<float4*>(mom);
    float4* s4 = reinterpret_cast<float4*>(sq);
    float4* ref4 = reinterpret_cast<float4*>(anchor);
    float4* vel4 = reinterpret_cast<float4*>(slow_v);
    for (int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; c < nq;
         c += (int64_t)gridDim.x * blockDim.x) {
        float4 gv[WMAX], th[WMAX], bu[WMAX], sv[WMAX], ref, vel;
#pragma unroll
        for (int k = 0; k < WMAX; ++k) {
            if (k < W) {
                const int64_t e = CPDP_IDX((int64_t)k * nq + c, (int64_t)W * nq);
                gv[k] = GradLoad<G>::vec4(grads, e);
                th[k] = p4[e];
                bu[k] = m4[e];
                if (OPT == kOptAdamW) sv[k] = s4[e];
            }
        }
        if (METHOD == kMethodCPDP) {
            ref = ref4[CPDP_IDX(c, nq)];
            vel = vel4[CPDP_IDX(c, nq)];
        }
        // 1. gradient mean (eq. 2)
        float4 gbar = make_float4(0.f, 0.f, 0.f, 0.f);
        if (METHOD != kMethodLocalSGD) {
            float4 gsum = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
            for (int k = 0; k < WMAX; ++k)
                if (k < W) add4(gsum, gv[k]);
            gbar = div4(gsum, a.workers);
        }
        // 2-3. optimizer step on every worker, then the mean of the stepped replicas (eq. 7)
        float4 tsum = make_float4(0.f, 0.f, 0.f, 0.f);
        float4 bsum = make_float4(0.f, 0.f, 0.f, 0.f), ssum = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int k = 0; k < WMAX; ++k) {
            if (k < W) {
                const int64_t e = CPDP_IDX((int64_t)k * nq + c, (int64_t)W * nq);
                opt_step4<OPT>(METHOD == kMethodLocalSGD ? gv[k] : gbar, th[k], bu[k], sv[k], a.step);
                if (STATE_SYNC) {
                    add4(bsum, bu[k]);
                    if (OPT == kOptAdamW) add4(ssum, sv[k]);
                } else {
                    m4[e] = bu[k];
                    if (OPT == kOptAdamW) s4[e] = sv[k];
                }
                if (METHOD == kMethodDDP)
                    p4[e] = th[k];
                else
                    add4(tsum, th[k]);
            }
        }
        if (METHOD == kMethodDDP) continue;
        if (STATE_SYNC) {
            const float4 bmean = div4(bsum, a.workers);
            const float4 smean = div4(ssum, a.workers);
#pragma unroll
            for (int k = 0; k < WMAX; ++k) {
                if (k < W) {
                    const int64_t e = CPDP_IDX((int64_t)k * nq + c, (int64_t)W * nq);
                    m4[e] = bmean;
                    if (OPT == kOptAdamW) s4[e] = smean;
                }
            }
        }
        const float4 avg = div4(tsum, a.workers);
        // 4. SlowMo (eqs. 8-10); LocalSGD writes the plain average
        float4 tn = avg;
        if (METHOD == kMethodCPDP) {
            float4 vn;
            vn.x = fmaf(a.beta, vel.x, avg.x - ref.x);
            vn.y = fmaf(a.beta, vel.y, avg.y - ref.y);
            vn.z = fmaf(a.beta, vel.z, avg.z - ref.z);
            vn.w = fmaf(a.beta, vel.w, avg.w - ref.w);
            tn.x = fmaf(a.alpha, vn.x, ref.x);
            tn.y = fmaf(a.alpha, vn.y, ref.y);
            tn.z = fmaf(a.alpha, vn.z, ref.z);
            tn.w = fmaf(a.alpha, vn.w, ref.w);
            ref4[CPDP_IDX(c, nq)] = tn;
            vel4[CPDP_IDX(c, nq)] = vn;
        }
        // 5. write-back to every replica (eqs. 11-12)
#pragma unroll
        for (int k = 0; k < WMAX; ++k)
            if (k < W) p4[CPDP_IDX((int64_t)k * nq + c, (int64_t)W * nq)] = tn;
    }
}

// Same computation, one parameter per thread, for any N (rows need not be
// 16-byte aligned).
template <int METHOD, int OPT, bool STATE_SYNC, typename G>
__global__ void __launch_bounds__(kThreads)
reconcile_scalar_kernel(float* __restrict__ params, float* __restrict__ mom, float* __restrict__ sq,
                        const G* __restrict__ grads, float* __restrict__ anchor, float* __restrict__ slow_v,
                        int W, int64_t N, SyncArgs a) {
    static_assert(!(STATE_SYNC && METHOD == kMethodDDP), "DDP's states are identical across workers");
    pdl_wait_then_release();
    for (int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; j < N;
         j += (int64_t)gridDim.x * blockDim.x) {
        float gbar = 0.f;
        if (METHOD != kMethodLocalSGD) {
            float gsum = 0.f;
            for (int i = 0; i < W; ++i) gsum += GradLoad<G>::one(grads, CPDP_IDX((int64_t)i * N + j, (int64_t)W * N));
            gbar = gsum / a.workers;
        }
        float tsum = 0.f, bsum = 0.f, ssum = 0.f;
        for (int i = 0; i < W; ++i) {
            float th = params[CPDP_IDX((int64_t)i * N + j, (int64_t)W * N)];
            float bu = mom[CPDP_IDX((int64_t)i * N + j, (int64_t)W * N)];
            float sv = 0.f;
            if (OPT == kOptAdamW) sv = sq[CPDP_IDX((int64_t)i * N + j, (int64_t)W * N)];
            const float g = METHOD == kMethodLocalSGD ? GradLoad<G>::one(grads, CPDP_IDX((int64_t)i * N + j, (int64_t)W * N)) : gbar;
            opt_step<OPT>(g, th, bu, sv, a.step);
            if (STATE_SYNC) {
                bsum += bu;
                ssum += sv;
            } else {
                mom[CPDP_IDX((int64_t)i * N + j, (int64_t)W * N)] = bu;
                if (OPT == kOptAdamW) sq[CPDP_IDX((int64_t)i * N + j, (int64_t)W * N)] = sv;
            }
            if (METHOD == kMethodDDP)
                params[CPDP_IDX((int64_t)i * N + j, (int64_t)W * N)] = th;
            else
                tsum += th;
        }
        if (METHOD == kMethodDDP) continue;
        if (STATE_SYNC) {
            const float bmean = bsum / a.workers, smean = ssum / a.workers;
            for (int i = 0; i < W; ++i) {
                mom[CPDP_IDX((int64_t)i * N + j, (int64_t)W * N)] = bmean;
                if (OPT == kOptAdamW) sq[CPDP_IDX((int64_t)i * N + j, (int64_t)W * N)] = smean;
            }
        }
        const float avg = tsum / a.workers;
        float tn = avg;
        if (METHOD == kMethodCPDP) {
            const float ref = anchor[CPDP_IDX(j, N)];
            const float vn = fmaf(a.beta, slow_v[CPDP_IDX(j, N)], avg - ref);
            tn = fmaf(a.alpha, vn, ref);
            anchor[CPDP_IDX(j, N)] = tn;
            slow_v[CPDP_IDX(j, N)] = vn;
        }
        for (int i = 0; i < W; ++i) params[CPDP_IDX((int64_t)i * N + j, (int64_t)W * N)] = tn;
    }
}

}  // namespace cpdp
