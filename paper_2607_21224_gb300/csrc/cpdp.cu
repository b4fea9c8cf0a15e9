// libcpdp: C ABI (include/cpdp.h) over the CPDP hot-path kernels.
//
// Host side only: argument validation, the context, the synchronization
// schedule (eq. 4 with the epoch-end rule of Sec. 3.1) and kernel launches.
// Every step of the path itself runs in the kernels of cpdp_kernels.cuh.
#include "cpdp.h"
#include "cpdp_floor.cuh"
#include "cpdp_kernels.cuh"
#include "cpdp_shapes.cuh"
#include "cpdp_shuffle.cuh"
#include "cpdp_tma.cuh"

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <new>
#include <string>
#include <type_traits>
#include <unordered_set>
#include <vector>

namespace {

constexpr uint64_t kMagic = 0x43504450636f6e74ull;  // "CPDPcont"
constexpr int kMaxWorkers = 4096;

thread_local std::string t_error;  // errors of calls without a usable context

std::mutex g_live_mutex;
std::unordered_set<const cpdp_ctx*>& live_contexts() {
    static std::unordered_set<const cpdp_ctx*> s;
    return s;
}

}  // namespace

struct cpdp_ctx {
    uint64_t magic = kMagic;
    int W = 0;
    int64_t N = 0;
    std::vector<int64_t> offsets;
    float lr = 0.f, momentum = 0.f, weight_decay = 0.f, beta = 0.f, alpha = 1.f;
    int K = 1;
    float* params = nullptr;
    float* mom = nullptr;
    float* anchor = nullptr;
    float* slow_v = nullptr;
    int device = -1;
    cpdp_method method = CPDP_METHOD_CPDP;
    // workers' optimizer: SGD with momentum (default) or AdamW (cpdp_set_adamw)
    cpdp_optimizer optimizer = CPDP_OPT_SGD;
    float adam_beta1 = 0.9f, adam_beta2 = 0.999f, adam_eps = 1e-8f;
    float* exp_avg_sq = nullptr;  // caller-owned [W][N], AdamW second moments
    int64_t opt_step = 0;         // optimizer steps taken (AdamW bias correction)
    bool state_sync = false;      // optimizer-state reconciliation variant
    bool pdl = true;              // programmatic dependent launches (cpdp_set_pdl)
    // reconcile rows staged through shared memory by bulk copies (cpdp_set_reconcile_staging):
    // 0 = off (direct loads), else the ring's slot count, with the launch's shared memory and grid
    int tma_stages = 0;
    size_t tma_smem = 0;
    unsigned tma_grid = 0;
    int64_t tma_withheld_tile = -1;  // cpdp_withhold_staged_tile: for the next staged reconcile only
    // reconcile with worker rows split across a warp's lanes and shuffle sums (cpdp_set_reconcile_shuffle)
    bool shuffle = false;
    const char* reconcile_kernel = "";  // the kernel the last reconcile launched (cpdp_reconcile_kernel)
    // collective-equivalents performed since creation (Table 2's counts)
    int64_t grad_means = 0, param_means = 0;
    // training-protocol schedule (cpdp_set_schedule)
    bool has_schedule = false;
    int64_t sched_steps = 0, sched_epochs = 0, sched_warmup = 0;
    float sched_base_lr = 0.f, sched_min_lr = 0.f;
    // gradient buffers whose memory type was already checked (a small ring), so
    // that steady-state calls, and calls made while a CUDA graph is being
    // captured after one eager call per buffer, make no pointer query
    static constexpr int kCheckedSlots = 16;
    const void* checked_grads[kCheckedSlots] = {};
    int checked_next = 0;
    // host-fed gradients (cpdp_bind_staging / cpdp_step_host): two caller-owned
    // device staging buffers, and the library's copy stream and events
    void* staging[2] = {nullptr, nullptr};
    size_t staging_bytes = 0;
    cudaStream_t copy_stream = nullptr;
    cudaEvent_t copied[2] = {nullptr, nullptr};
    cudaEvent_t consumed[2] = {nullptr, nullptr};
    bool staging_used[2] = {false, false};
    int64_t staged = 0;
    std::string error;
};

namespace {

cpdp_status set_error(cpdp_ctx* ctx, cpdp_status st, const char* fmt, ...) {
    char msg[512];
    va_list ap;
    va_start(ap, fmt);
    std::vsnprintf(msg, sizeof msg, fmt, ap);
    va_end(ap);
    if (ctx != nullptr)
        ctx->error = msg;
    else
        t_error = msg;
    return st;
}

// A pointer is usable only while it is a live context (created and not yet
// destroyed); a stale or foreign pointer is rejected without being read.
bool usable(const cpdp_ctx* ctx) {
    if (ctx == nullptr) return false;
    std::lock_guard<std::mutex> lock(g_live_mutex);
    return live_contexts().count(ctx) != 0 && ctx->magic == kMagic;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

bool overlaps(const void* a, size_t na, const void* b, size_t nb) {
    const uintptr_t a0 = reinterpret_cast<uintptr_t>(a), b0 = reinterpret_cast<uintptr_t>(b);
    return a0 < b0 + nb && b0 < a0 + na;
}

size_t row_bytes(const cpdp_ctx* c) { return static_cast<size_t>(c->N) * sizeof(float); }
size_t state_bytes(const cpdp_ctx* c) { return static_cast<size_t>(c->W) * row_bytes(c); }

// The bound state ranges, for overlap checks against other buffers.
bool overlaps_state(const cpdp_ctx* c, const void* p, size_t n) {
    return overlaps(p, n, c->params, state_bytes(c)) || overlaps(p, n, c->mom, state_bytes(c)) ||
           overlaps(p, n, c->anchor, row_bytes(c)) || overlaps(p, n, c->slow_v, row_bytes(c)) ||
           (c->exp_avg_sq != nullptr && overlaps(p, n, c->exp_avg_sq, state_bytes(c)));
}

// Optimizer scalars for the step with 1-based count `step`; AdamW's bias
// corrections and decoupled decay factor are formed in double precision.
cpdp::StepArgs step_args(const cpdp_ctx* c, int64_t step) {
    cpdp::StepArgs a{};
    a.lr = c->lr;
    a.momentum = c->momentum;
    a.weight_decay = c->weight_decay;
    if (c->optimizer == CPDP_OPT_ADAMW) {
        const double lr = c->lr, wd = c->weight_decay, b1 = c->adam_beta1, b2 = c->adam_beta2;
        const double bc1 = 1.0 - std::pow(b1, static_cast<double>(step));
        const double bc2 = 1.0 - std::pow(b2, static_cast<double>(step));
        a.adam.decay = static_cast<float>(1.0 - lr * wd);
        a.adam.step_size = static_cast<float>(lr / bc1);
        a.adam.inv_bc2_sqrt = static_cast<float>(1.0 / std::sqrt(bc2));
        a.adam.beta1 = c->adam_beta1;
        a.adam.one_minus_beta1 = static_cast<float>(1.0 - b1);
        a.adam.beta2 = c->adam_beta2;
        a.adam.one_minus_beta2 = static_cast<float>(1.0 - b2);
        a.adam.eps = c->adam_eps;
    }
    return a;
}

cpdp_status cuda_fail(cpdp_ctx* ctx, cudaError_t e, const char* what) {
    return set_error(ctx, CPDP_ECUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

// Make the context's device current (the caller may have switched devices).
cpdp_status enter_device(cpdp_ctx* ctx) {
    int cur = -1;
    cudaError_t e = cudaGetDevice(&cur);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaGetDevice");
    if (cur != ctx->device) {
        e = cudaSetDevice(ctx->device);
        if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaSetDevice");
    }
    return CPDP_OK;
}

// The result of a launch: its own error, else any error the runtime recorded.
cpdp_status check_launch(cpdp_ctx* ctx, cudaError_t launched, const char* what) {
    const cudaError_t e = launched != cudaSuccess ? launched : cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(ctx, e, what);
    return CPDP_OK;
}

// Launch `kernel` with kThreads threads per block on `s`. With the context's
// programmatic dependent launch on, the launch may begin while the previous
// grid on the stream drains; every kernel waits for that grid's completion
// itself before touching memory (cpdp::pdl_wait_then_release).
template <typename... KArgs, typename... Args>
cudaError_t launch_shaped(bool pdl, void (*kernel)(KArgs...), unsigned grid, unsigned block, size_t smem,
                          cudaStream_t s, Args... args) {
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(block);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kernel, args...);
}

template <typename... KArgs, typename... Args>
cudaError_t launch(const cpdp_ctx* c, void (*kernel)(KArgs...), unsigned grid, cudaStream_t s, Args... args) {
    return launch_shaped(c->pdl, kernel, grid, cpdp::kThreads, 0, s, args...);
}

// Whether `s` is being captured into a CUDA graph (a query that is legal
// during capture).
cpdp_status capture_active(cpdp_ctx* ctx, cudaStream_t s, bool* active) {
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    const cudaError_t e = cudaStreamIsCapturing(s, &cs);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaStreamIsCapturing");
    *active = cs != cudaStreamCaptureStatusNone;
    return CPDP_OK;
}

// Refuse a call under capture when a replay would repeat a stale argument.
cpdp_status refuse_capture(cpdp_ctx* ctx, cudaStream_t s, const char* why) {
    bool active = false;
    const cpdp_status st = capture_active(ctx, s, &active);
    if (st != CPDP_OK) return st;
    if (active) return set_error(ctx, CPDP_ESTATE, "cannot be captured into a CUDA graph: %s", why);
    return CPDP_OK;
}

// An input the kernels read: device or managed memory on the context's
// device, or page-locked host memory (reachable from the GPU); pageable host
// memory is refused.
cpdp_status check_readable(cpdp_ctx* ctx, const void* p, const char* what) {
    cudaPointerAttributes at;
    const cudaError_t e = cudaPointerGetAttributes(&at, p);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaPointerGetAttributes");
    if (at.type == cudaMemoryTypeUnregistered)
        return set_error(ctx, CPDP_EINVAL, "%s %p is pageable host memory; pass device or page-locked memory", what, p);
    if (at.type == cudaMemoryTypeDevice && at.device != ctx->device)
        return set_error(ctx, CPDP_EINVAL, "%s lives on device %d, state on device %d", what, at.device, ctx->device);
    return CPDP_OK;
}

// Shared checks of the gradient argument of the step entry points.
cpdp_status check_grads(cpdp_ctx* ctx, const void* grads, cpdp_dtype dtype) {
    if (ctx->params == nullptr) return set_error(ctx, CPDP_ESTATE, "state buffers not bound (call cpdp_bind first)");
    if (grads == nullptr) return set_error(ctx, CPDP_EINVAL, "grads is NULL");
    if (dtype != CPDP_F32 && dtype != CPDP_BF16) return set_error(ctx, CPDP_EINVAL, "unknown gradient dtype %d", (int)dtype);
    if (!aligned16(grads)) return set_error(ctx, CPDP_EALIGN, "grads %p is not 16-byte aligned", grads);
    const size_t elt = dtype == CPDP_F32 ? sizeof(float) : sizeof(uint16_t);
    const size_t gbytes = static_cast<size_t>(ctx->W) * static_cast<size_t>(ctx->N) * elt;
    if (overlaps_state(ctx, grads, gbytes)) return set_error(ctx, CPDP_EINVAL, "grads overlap the bound state buffers");
    for (const void* p : ctx->checked_grads)
        if (p == grads) return CPDP_OK;
    const cpdp_status st = check_readable(ctx, grads, "grads");
    if (st != CPDP_OK) return st;
    ctx->checked_grads[ctx->checked_next] = grads;
    ctx->checked_next = (ctx->checked_next + 1) % cpdp_ctx::kCheckedSlots;
    return CPDP_OK;
}

template <typename G>
cudaError_t launch_local(cpdp_ctx* c, const void* grads, cudaStream_t s, const cpdp::StepArgs& a) {
    const int64_t total = static_cast<int64_t>(c->W) * c->N;
    const int64_t nq = total >> 2;
    const unsigned grid = cpdp::grid_for(nq > 0 ? nq : 1, (int64_t)cpdp::kThreads * cpdp::kLocalUnroll);
    const G* g = static_cast<const G*>(grads);
    if (c->optimizer == CPDP_OPT_ADAMW)
        return launch(c,
                      cpdp::local_step_kernel<cpdp::kOptAdamW, G, cpdp::kLocalUnroll,
                                              cpdp::LocalWarpRuns<cpdp::kOptAdamW, G>::value>,
                      grid, s, c->params, c->mom, c->exp_avg_sq, g, total, a);
    return launch(c,
                  cpdp::local_step_kernel<cpdp::kOptSGD, G, cpdp::kLocalUnroll, cpdp::LocalWarpRuns<cpdp::kOptSGD, G>::value>,
                  grid, s, c->params, c->mom, static_cast<float*>(nullptr), g, total, a);
}

// The one-pass reconcile for at most Shape::wmax workers.
template <typename Shape, int METHOD, int OPT, bool SS, typename G>
cudaError_t launch_onepass(cpdp_ctx* c, const G* g, float* sq, cudaStream_t s, const cpdp::SyncArgs& a, int64_t nq) {
    static_assert(Shape::use, "a one-pass shape that is not used");
    c->reconcile_kernel = "reconcile_onepass_kernel";
    return launch(c, cpdp::reconcile_onepass_kernel<METHOD, OPT, SS, G, Shape::wmax, Shape::min_blocks>,
                  cpdp::grid_for(nq, cpdp::kThreads), s, c->params, c->mom, sq, g, c->anchor, c->slow_v, c->W, nq, a);
}

// The vectorised reconcile in launch shape Shape, with 32-bit offsets where
// the shape asks for them and the sizes allow.
template <typename Shape, int METHOD, int OPT, bool SS, typename G>
cudaError_t launch_vec4(cpdp_ctx* c, const G* g, float* sq, cudaStream_t s, const cpdp::SyncArgs& a, int64_t nq) {
    const unsigned grid = cpdp::grid_for(nq, cpdp::kThreads);
    c->reconcile_kernel = "reconcile_vec4_kernel";
    constexpr int grad_rows = cpdp::GradChunkOf<Shape>::rows;
    constexpr bool overlap = cpdp::GradChunkOf<Shape>::overlap;
    if constexpr (Shape::narrow) {
        if (static_cast<int64_t>(c->W) * nq + static_cast<int64_t>(grid) * cpdp::kThreads < (int64_t(1) << 31))
            return launch(c,
                          cpdp::reconcile_vec4_kernel<METHOD, OPT, SS, G, Shape::rows, Shape::min_blocks, Shape::late,
                                                      int32_t, grad_rows, overlap>,
                          grid, s, c->params, c->mom, sq, g, c->anchor, c->slow_v, c->W, static_cast<int32_t>(nq), a);
    }
    return launch(c,
                  cpdp::reconcile_vec4_kernel<METHOD, OPT, SS, G, Shape::rows, Shape::min_blocks, Shape::late, int64_t,
                                              grad_rows, overlap>,
                  grid, s, c->params, c->mom, sq, g, c->anchor, c->slow_v, c->W, nq, a);
}

template <int METHOD, int OPT, bool SS, typename G>
cudaError_t launch_reconcile_variant(cpdp_ctx* c, const void* grads, cudaStream_t s, const cpdp::StepArgs& step) {
    const cpdp::SyncArgs a{step, c->beta, c->alpha, static_cast<float>(c->W)};
    float* sq = OPT == cpdp::kOptAdamW ? c->exp_avg_sq : nullptr;
    const G* g = static_cast<const G*>(grads);
    if ((c->N & 3) == 0) {
        const int64_t nq = c->N >> 2;
        // few workers: one round trip where it measured faster (cpdp_shapes.cuh)
        if (c->W == 1) return launch_onepass<cpdp::OnePassW1, METHOD, OPT, SS, G>(c, g, sq, s, a, nq);
        using P2 = cpdp::OnePassW2<METHOD, OPT, SS, G>;
        using P3 = cpdp::OnePassW3<METHOD, OPT, SS, G>;
        using P4 = cpdp::OnePassW4<METHOD, OPT, SS, G>;
        if constexpr (P2::use)
            if (c->W == 2) return launch_onepass<P2, METHOD, OPT, SS, G>(c, g, sq, s, a, nq);
        if constexpr (P3::use)
            if (c->W == 3) return launch_onepass<P3, METHOD, OPT, SS, G>(c, g, sq, s, a, nq);
        if constexpr (P4::use)
            if (c->W == 4) return launch_onepass<P4, METHOD, OPT, SS, G>(c, g, sq, s, a, nq);
        using T3 = cpdp::ReconcileThreeRows<METHOD, OPT, SS, G, 3>;
        using T5 = cpdp::ReconcileThreeRows<METHOD, OPT, SS, G, 5>;
        using T6 = cpdp::ReconcileThreeRows<METHOD, OPT, SS, G, 6>;
        if constexpr (T3::use)
            if (c->W == 3) return launch_vec4<T3, METHOD, OPT, SS, G>(c, g, sq, s, a, nq);
        if constexpr (T5::use)
            if (c->W == 5) return launch_vec4<T5, METHOD, OPT, SS, G>(c, g, sq, s, a, nq);
        if constexpr (T6::use)
            if (c->W == 6) return launch_vec4<T6, METHOD, OPT, SS, G>(c, g, sq, s, a, nq);
        using GCFew = cpdp::ReconcileGradChunks<METHOD, OPT, SS, G, false>;
        using GCMany = cpdp::ReconcileGradChunks<METHOD, OPT, SS, G, true>;
        if constexpr (GCMany::use)
            if (c->W >= cpdp::kGradChunksManyWorkers) return launch_vec4<GCMany, METHOD, OPT, SS, G>(c, g, sq, s, a, nq);
        if constexpr (GCFew::use)
            if (c->W >= GCFew::min_workers && c->W <= GCFew::max_workers)
                return launch_vec4<GCFew, METHOD, OPT, SS, G>(c, g, sq, s, a, nq);
        if (c->W >= 3 && c->W <= 6)
            return launch_vec4<cpdp::ReconcileShapeFew<OPT, G, SS>, METHOD, OPT, SS, G>(c, g, sq, s, a, nq);
        if (c->W == 2) return launch_vec4<cpdp::ReconcileShapeW2<OPT, G, SS>, METHOD, OPT, SS, G>(c, g, sq, s, a, nq);
        return launch_vec4<cpdp::ReconcileShape<OPT, G, SS>, METHOD, OPT, SS, G>(c, g, sq, s, a, nq);
    }
    c->reconcile_kernel = "reconcile_scalar_kernel";
    return launch(c, cpdp::reconcile_scalar_kernel<METHOD, OPT, SS, G>, cpdp::grid_for(c->N, cpdp::kThreads), s, c->params,
                  c->mom, sq, g, c->anchor, c->slow_v, c->W, c->N, a);
}

template <int METHOD, int OPT, typename G>
cudaError_t launch_reconcile_state(cpdp_ctx* c, const void* grads, cudaStream_t s, const cpdp::StepArgs& a) {
    if (c->state_sync) return launch_reconcile_variant<METHOD, OPT, true, G>(c, grads, s, a);
    return launch_reconcile_variant<METHOD, OPT, false, G>(c, grads, s, a);
}

template <int OPT, typename G>
cudaError_t launch_reconcile_opt(cpdp_ctx* c, const void* grads, cudaStream_t s, const cpdp::StepArgs& a) {
    switch (c->method) {
        case CPDP_METHOD_LOCALSGD:
            return launch_reconcile_state<cpdp::kMethodLocalSGD, OPT, G>(c, grads, s, a);
        case CPDP_METHOD_DDP:  // states are identical across workers: nothing to reconcile
            return launch_reconcile_variant<cpdp::kMethodDDP, OPT, false, G>(c, grads, s, a);
        default:
            return launch_reconcile_state<cpdp::kMethodCPDP, OPT, G>(c, grads, s, a);
    }
}

template <typename G>
cudaError_t launch_reconcile(cpdp_ctx* c, const void* grads, cudaStream_t s, const cpdp::StepArgs& a) {
    if (c->optimizer == CPDP_OPT_ADAMW) return launch_reconcile_opt<cpdp::kOptAdamW, G>(c, grads, s, a);
    return launch_reconcile_opt<cpdp::kOptSGD, G>(c, grads, s, a);
}

cudaError_t launch_reconcile_tma(cpdp_ctx* c, const float* grads, cudaStream_t s, const cpdp::StepArgs& step) {
    const cpdp::SyncArgs a{step, c->beta, c->alpha, static_cast<float>(c->W)};
    const int64_t ntiles = (c->N + cpdp::kTmaTile - 1) / cpdp::kTmaTile;
    const unsigned grid = static_cast<unsigned>(ntiles < (int64_t)c->tma_grid ? ntiles : c->tma_grid);
    const int64_t withheld = c->tma_withheld_tile;
    c->tma_withheld_tile = -1;
    c->reconcile_kernel = "reconcile_tma_kernel";
    return launch_shaped(c->pdl, cpdp::reconcile_tma_kernel, grid, cpdp::kTmaThreads, c->tma_smem, s, c->params,
                         c->mom, grads, c->anchor, c->slow_v, c->W, c->N, c->tma_stages, withheld, a);
}

cudaError_t launch_reconcile_shuffle(cpdp_ctx* c, const float* grads, cudaStream_t s, const cpdp::StepArgs& step) {
    const cpdp::SyncArgs a{step, c->beta, c->alpha, static_cast<float>(c->W)};
    const int64_t nq = c->N >> 2;
    const int64_t tiles = (nq + cpdp::kShuffleCols - 1) / cpdp::kShuffleCols;
    c->reconcile_kernel = "reconcile_shuffle_kernel";
    return launch(c, cpdp::reconcile_shuffle_kernel, cpdp::grid_for(tiles, cpdp::kThreads / 32), s, c->params, c->mom,
                  grads, c->anchor, c->slow_v, c->W, nq, a);
}

// The column-walk floor (cpdp_floor_columns) in one of its compiled shapes.
template <typename G, int CH, int MB>
cudaError_t launch_floor_columns(float* params, float* mom, float* sq, const void* grads, float* anchor, float* slow_v,
                                 int W, int64_t nq, cudaStream_t s) {
    return launch_shaped(true, cpdp::floor_columns_kernel<G, CH, MB>, cpdp::grid_for(nq, cpdp::kThreads),
                         cpdp::kThreads, 0, s, params, mom, sq, static_cast<const G*>(grads), anchor, slow_v, W, nq);
}

template <typename G>
cudaError_t launch_floor_columns_shape(int chunk_rows, int blocks, float* params, float* mom, float* sq,
                                       const void* grads, float* anchor, float* slow_v, int W, int64_t nq,
                                       cudaStream_t s) {
    if (chunk_rows == 2) return launch_floor_columns<G, 2, 4>(params, mom, sq, grads, anchor, slow_v, W, nq, s);
    if (chunk_rows == 3) return launch_floor_columns<G, 3, 3>(params, mom, sq, grads, anchor, slow_v, W, nq, s);
    return launch_floor_columns<G, 4, 2>(params, mom, sq, grads, anchor, slow_v, W, nq, s);
}


static_assert(cpdp::kMethodCPDP == CPDP_METHOD_CPDP && cpdp::kMethodLocalSGD == CPDP_METHOD_LOCALSGD &&
                  cpdp::kMethodDDP == CPDP_METHOD_DDP,
              "kernel method tags follow the ABI's cpdp_method values");
static_assert(cpdp::kOptSGD == CPDP_OPT_SGD && cpdp::kOptAdamW == CPDP_OPT_ADAMW,
              "kernel optimizer tags follow the ABI's cpdp_optimizer values");

bool finite_all(std::initializer_list<float> xs) {
    for (float x : xs)
        if (!std::isfinite(x)) return false;
    return true;
}

}  // namespace

extern "C" {

cpdp_status cpdp_create(cpdp_ctx** out, int W, int64_t N, const int64_t* tensor_offsets, int num_tensors,
                        float lr, float momentum, float weight_decay, int K, float slowmo_beta,
                        float slowmo_alpha) {
    if (out == nullptr) return set_error(nullptr, CPDP_EINVAL, "out is NULL");
    *out = nullptr;
    if (W < 1 || W > kMaxWorkers) return set_error(nullptr, CPDP_EINVAL, "W=%d outside [1, %d]", W, kMaxWorkers);
    if (N < 1) return set_error(nullptr, CPDP_EINVAL, "N=%lld must be >= 1", (long long)N);
    if (N > (int64_t(1) << 40) / W) return set_error(nullptr, CPDP_EINVAL, "W*N too large");
    if (!finite_all({lr, momentum, weight_decay, slowmo_beta, slowmo_alpha}))
        return set_error(nullptr, CPDP_EINVAL, "hyperparameters must be finite");
    if (!(lr > 0.f)) return set_error(nullptr, CPDP_EINVAL, "lr=%g must be > 0", (double)lr);
    if (momentum < 0.f) return set_error(nullptr, CPDP_EINVAL, "momentum=%g must be >= 0", (double)momentum);
    if (weight_decay < 0.f) return set_error(nullptr, CPDP_EINVAL, "weight_decay=%g must be >= 0", (double)weight_decay);
    if (K < 1) return set_error(nullptr, CPDP_EINVAL, "K=%d must be >= 1", K);
    if (!(slowmo_beta >= 0.f && slowmo_beta < 1.f))
        return set_error(nullptr, CPDP_EINVAL, "slowmo_beta=%g outside [0, 1)", (double)slowmo_beta);
    if (!(slowmo_alpha > 0.f)) return set_error(nullptr, CPDP_EINVAL, "slowmo_alpha=%g must be > 0", (double)slowmo_alpha);
    if (num_tensors < 0) return set_error(nullptr, CPDP_EINVAL, "num_tensors=%d < 0", num_tensors);
    if (num_tensors > 0 && tensor_offsets == nullptr)
        return set_error(nullptr, CPDP_EINVAL, "tensor_offsets is NULL with num_tensors=%d", num_tensors);
    if (num_tensors > 0) {
        if (tensor_offsets[0] != 0) return set_error(nullptr, CPDP_EINVAL, "tensor_offsets[0]=%lld must be 0", (long long)tensor_offsets[0]);
        for (int k = 0; k < num_tensors; ++k) {
            if (tensor_offsets[k + 1] <= tensor_offsets[k])
                return set_error(nullptr, CPDP_EINVAL, "tensor_offsets not strictly increasing at %d", k);
        }
        if (tensor_offsets[num_tensors] != N)
            return set_error(nullptr, CPDP_EINVAL, "tensor_offsets[%d]=%lld must equal N=%lld", num_tensors,
                             (long long)tensor_offsets[num_tensors], (long long)N);
    }
    cpdp_ctx* c = new (std::nothrow) cpdp_ctx();
    if (c == nullptr) return set_error(nullptr, CPDP_ENOMEM, "out of host memory");
    try {
        if (num_tensors > 0)
            c->offsets.assign(tensor_offsets, tensor_offsets + num_tensors + 1);
        else
            c->offsets = {0, N};
        std::lock_guard<std::mutex> lock(g_live_mutex);
        live_contexts().insert(c);
    } catch (...) {
        delete c;
        return set_error(nullptr, CPDP_ENOMEM, "out of host memory");
    }
    c->W = W;
    c->N = N;
    c->lr = lr;
    c->momentum = momentum;
    c->weight_decay = weight_decay;
    c->K = K;
    c->beta = slowmo_beta;
    c->alpha = slowmo_alpha;
    *out = c;
    return CPDP_OK;
}

cpdp_status cpdp_bind(cpdp_ctx* ctx, float* params, float* mom, float* anchor, float* slow_v) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    if (!params || !mom || !anchor || !slow_v) return set_error(ctx, CPDP_EINVAL, "a state pointer is NULL");
    if (!aligned16(params) || !aligned16(mom) || !aligned16(anchor) || !aligned16(slow_v))
        return set_error(ctx, CPDP_EALIGN, "state pointers must be 16-byte aligned");
    const size_t sb = state_bytes(ctx), rb = row_bytes(ctx);
    if (overlaps(params, sb, mom, sb) || overlaps(params, sb, anchor, rb) || overlaps(params, sb, slow_v, rb) ||
        overlaps(mom, sb, anchor, rb) || overlaps(mom, sb, slow_v, rb) || overlaps(anchor, rb, slow_v, rb))
        return set_error(ctx, CPDP_EINVAL, "state buffers overlap");
    int device = -1;
    const float* ptrs[4] = {params, mom, anchor, slow_v};
    for (const float* p : ptrs) {
        cudaPointerAttributes at;
        const cudaError_t e = cudaPointerGetAttributes(&at, p);
        if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaPointerGetAttributes(state)");
        if (at.type != cudaMemoryTypeDevice && at.type != cudaMemoryTypeManaged)
            return set_error(ctx, CPDP_EINVAL, "state pointer %p is not device memory", (const void*)p);
        if (device < 0) device = at.device;
        if (at.device != device) return set_error(ctx, CPDP_EINVAL, "state buffers live on different devices");
    }
    ctx->params = params;
    ctx->mom = mom;
    ctx->anchor = anchor;
    ctx->slow_v = slow_v;
    ctx->device = device;
    for (const void*& p : ctx->checked_grads) p = nullptr;
    return enter_device(ctx);
}

cpdp_status cpdp_init_params(cpdp_ctx* ctx, const float* theta0, void* stream) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    if (ctx->params == nullptr) return set_error(ctx, CPDP_ESTATE, "state buffers not bound (call cpdp_bind first)");
    if (theta0 == nullptr) return set_error(ctx, CPDP_EINVAL, "theta0 is NULL");
    if (!aligned16(theta0)) return set_error(ctx, CPDP_EALIGN, "theta0 is not 16-byte aligned");
    if (overlaps_state(ctx, theta0, row_bytes(ctx))) return set_error(ctx, CPDP_EINVAL, "theta0 overlaps the state buffers");
    cpdp_status st = check_readable(ctx, theta0, "theta0");
    if (st != CPDP_OK) return st;
    if ((st = enter_device(ctx)) != CPDP_OK) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    float* sq = ctx->optimizer == CPDP_OPT_ADAMW ? ctx->exp_avg_sq : nullptr;
    cudaError_t e;
    if ((ctx->N & 3) == 0) {
        const int64_t nq = ctx->N >> 2;
        e = launch(ctx, cpdp::init_vec4_kernel, cpdp::grid_for(nq, cpdp::kThreads), s, ctx->params, ctx->mom, sq,
                   ctx->anchor, ctx->slow_v, theta0, ctx->W, nq);
    } else {
        e = launch(ctx, cpdp::init_scalar_kernel, cpdp::grid_for(ctx->N, cpdp::kThreads), s, ctx->params, ctx->mom, sq,
                   ctx->anchor, ctx->slow_v, theta0, ctx->W, ctx->N);
    }
    if ((st = check_launch(ctx, e, "init kernel launch")) != CPDP_OK) return st;
    ctx->opt_step = 0;
    return CPDP_OK;
}

cpdp_status cpdp_local_step(cpdp_ctx* ctx, const void* grads, cpdp_dtype dtype, void* stream) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    cpdp_status st = check_grads(ctx, grads, dtype);
    if (st != CPDP_OK) return st;
    if ((st = enter_device(ctx)) != CPDP_OK) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (ctx->optimizer == CPDP_OPT_ADAMW &&
        (st = refuse_capture(ctx, s, "AdamW's bias correction depends on the step count")) != CPDP_OK)
        return st;
    const int64_t step = ctx->opt_step + 1;
    const cpdp::StepArgs a = step_args(ctx, step);
    const cudaError_t e = dtype == CPDP_F32 ? launch_local<float>(ctx, grads, s, a)
                                            : launch_local<cpdp::bf16_bits>(ctx, grads, s, a);
    if ((st = check_launch(ctx, e, "local-step kernel launch")) != CPDP_OK) return st;
    ctx->opt_step = step;
    return CPDP_OK;
}

cpdp_status cpdp_reconcile(cpdp_ctx* ctx, const void* grads, cpdp_dtype dtype, void* stream) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    cpdp_status st = check_grads(ctx, grads, dtype);
    if (st != CPDP_OK) return st;
    if ((st = enter_device(ctx)) != CPDP_OK) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (ctx->optimizer == CPDP_OPT_ADAMW &&
        (st = refuse_capture(ctx, s, "AdamW's bias correction depends on the step count")) != CPDP_OK)
        return st;
    const int64_t step = ctx->opt_step + 1;
    const cpdp::StepArgs a = step_args(ctx, step);
    cudaError_t e;
    if (ctx->shuffle) {
        if (ctx->method != CPDP_METHOD_CPDP || ctx->optimizer != CPDP_OPT_SGD || ctx->state_sync || dtype != CPDP_F32)
            return set_error(ctx, CPDP_ESTATE,
                             "the shuffle reconcile covers only the CPDP method with momentum SGD, float32 gradients "
                             "and no state reconciliation (cpdp_set_reconcile_shuffle(ctx, 0) turns it off)");
        e = launch_reconcile_shuffle(ctx, static_cast<const float*>(grads), s, a);
    } else if (ctx->tma_stages > 0) {
        if (ctx->method != CPDP_METHOD_CPDP || ctx->optimizer != CPDP_OPT_SGD || ctx->state_sync || dtype != CPDP_F32)
            return set_error(ctx, CPDP_ESTATE,
                             "the shared-memory-staged reconcile covers only the CPDP method with momentum SGD, "
                             "float32 gradients and no state reconciliation (cpdp_set_reconcile_staging(ctx, 0) "
                             "turns it off)");
        e = launch_reconcile_tma(ctx, static_cast<const float*>(grads), s, a);
    } else {
        e = dtype == CPDP_F32 ? launch_reconcile<float>(ctx, grads, s, a)
                              : launch_reconcile<cpdp::bf16_bits>(ctx, grads, s, a);
    }
    if ((st = check_launch(ctx, e, "reconcile kernel launch")) != CPDP_OK) return st;
    ctx->opt_step = step;
    if (ctx->method != CPDP_METHOD_LOCALSGD) ++ctx->grad_means;
    if (ctx->method != CPDP_METHOD_DDP) ++ctx->param_means;
    return CPDP_OK;
}

int cpdp_is_sync_step(const cpdp_ctx* ctx, int64_t t, int64_t steps_per_epoch) {
    if (!usable(ctx) || t < 1 || t > steps_per_epoch) return -1;
    if (ctx->method == CPDP_METHOD_DDP) return 1;  // DDP synchronizes every step (K = 1)
    return (t % ctx->K == 0 || t == steps_per_epoch) ? 1 : 0;
}

cpdp_status cpdp_set_method(cpdp_ctx* ctx, cpdp_method method) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    if (method != CPDP_METHOD_CPDP && method != CPDP_METHOD_LOCALSGD && method != CPDP_METHOD_DDP)
        return set_error(ctx, CPDP_EINVAL, "unknown method %d", (int)method);
    ctx->method = method;
    return CPDP_OK;
}

cpdp_status cpdp_set_adamw(cpdp_ctx* ctx, float beta1, float beta2, float eps, float* exp_avg_sq) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    if (ctx->params == nullptr) return set_error(ctx, CPDP_ESTATE, "state buffers not bound (call cpdp_bind first)");
    if (!finite_all({beta1, beta2, eps}) || !(beta1 >= 0.f && beta1 < 1.f) || !(beta2 >= 0.f && beta2 < 1.f) ||
        eps < 0.f)
        return set_error(ctx, CPDP_EINVAL, "AdamW needs betas in [0, 1) and a finite eps >= 0");
    if (exp_avg_sq == nullptr) return set_error(ctx, CPDP_EINVAL, "exp_avg_sq is NULL");
    if (!aligned16(exp_avg_sq)) return set_error(ctx, CPDP_EALIGN, "exp_avg_sq is not 16-byte aligned");
    float* keep = ctx->exp_avg_sq;
    ctx->exp_avg_sq = nullptr;  // check against the other state only
    if (overlaps_state(ctx, exp_avg_sq, state_bytes(ctx))) {
        ctx->exp_avg_sq = keep;
        return set_error(ctx, CPDP_EINVAL, "exp_avg_sq overlaps the state buffers");
    }
    cudaPointerAttributes at;
    const cudaError_t e = cudaPointerGetAttributes(&at, exp_avg_sq);
    if (e != cudaSuccess) {
        ctx->exp_avg_sq = keep;
        return cuda_fail(ctx, e, "cudaPointerGetAttributes(exp_avg_sq)");
    }
    if ((at.type != cudaMemoryTypeDevice && at.type != cudaMemoryTypeManaged) || at.device != ctx->device) {
        ctx->exp_avg_sq = keep;
        return set_error(ctx, CPDP_EINVAL, "exp_avg_sq must be device memory on the state's device");
    }
    ctx->exp_avg_sq = exp_avg_sq;
    ctx->adam_beta1 = beta1;
    ctx->adam_beta2 = beta2;
    ctx->adam_eps = eps;
    ctx->optimizer = CPDP_OPT_ADAMW;
    ctx->opt_step = 0;
    return CPDP_OK;
}

cpdp_status cpdp_set_state_reconcile(cpdp_ctx* ctx, int enable) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    if (enable != 0 && enable != 1) return set_error(ctx, CPDP_EINVAL, "enable must be 0 or 1");
    ctx->state_sync = enable == 1;
    return CPDP_OK;
}

cpdp_status cpdp_set_pdl(cpdp_ctx* ctx, int enable) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    if (enable != 0 && enable != 1) return set_error(ctx, CPDP_EINVAL, "enable must be 0 or 1");
    ctx->pdl = enable == 1;
    return CPDP_OK;
}

cpdp_status cpdp_set_reconcile_staging(cpdp_ctx* ctx, int stages) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    if (ctx->params == nullptr) return set_error(ctx, CPDP_ESTATE, "state buffers not bound (call cpdp_bind first)");
    if (stages == 0) {
        ctx->tma_stages = 0;
        return CPDP_OK;
    }
    if (stages < 2 || stages > 8) return set_error(ctx, CPDP_EINVAL, "stages=%d: 0 (off) or 2..8", stages);
    if (ctx->shuffle)
        return set_error(ctx, CPDP_ESTATE, "the shuffle reconcile is on; turn it off before staging the rows");
    if (ctx->W > cpdp::kTmaMaxWorkers)
        return set_error(ctx, CPDP_EINVAL, "the staged reconcile holds at most %d workers' rows (W=%d)",
                         cpdp::kTmaMaxWorkers, ctx->W);
    if ((ctx->N & 3) != 0) return set_error(ctx, CPDP_EINVAL, "the staged reconcile needs N a multiple of 4");
    cpdp_status st = enter_device(ctx);
    if (st != CPDP_OK) return st;
    const size_t smem = static_cast<size_t>(stages) * (3 * ctx->W + 2) * cpdp::kTmaTile * sizeof(float) +
                        3 * static_cast<size_t>(stages) * sizeof(uint64_t);
    int optin = 0, sms = 0, occ = 0;
    cudaError_t e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, ctx->device);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, ctx->device);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaDeviceGetAttribute");
    if (smem > static_cast<size_t>(optin))
        return set_error(ctx, CPDP_EINVAL, "%d slots of %d row segments need %zu bytes of shared memory; a block has %d",
                         stages, 3 * ctx->W + 2, smem, optin);
    // the kernel's limit is raised to the block maximum (not to this context's
    // need), so contexts with other slot counts keep launching
    e = cudaFuncSetAttribute(cpdp::reconcile_tma_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, optin);
    if (e == cudaSuccess)
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, cpdp::reconcile_tma_kernel, cpdp::kTmaThreads, smem);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "staged reconcile set-up");
    if (occ < 1) return set_error(ctx, CPDP_EINVAL, "the staged reconcile does not fit on an SM with %d slots", stages);
    ctx->tma_stages = stages;
    ctx->tma_smem = smem;
    ctx->tma_grid = static_cast<unsigned>(sms * occ);
    return CPDP_OK;
}

cpdp_status cpdp_set_reconcile_shuffle(cpdp_ctx* ctx, int enable) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    if (enable != 0 && enable != 1) return set_error(ctx, CPDP_EINVAL, "enable must be 0 or 1");
    if (enable == 1) {
        if ((ctx->N & 3) != 0) return set_error(ctx, CPDP_EINVAL, "the shuffle reconcile needs N a multiple of 4");
        if (ctx->tma_stages > 0)
            return set_error(ctx, CPDP_ESTATE, "the reconcile's rows are staged; turn staging off before this");
    }
    ctx->shuffle = enable == 1;
    return CPDP_OK;
}

cpdp_status cpdp_withhold_staged_tile(cpdp_ctx* ctx, int64_t tile) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    if (ctx->tma_stages == 0) return set_error(ctx, CPDP_ESTATE, "the staged reconcile is off");
    const int64_t tiles = (ctx->N + cpdp::kTmaTile - 1) / cpdp::kTmaTile;
    if (tile < 0 || tile >= tiles)
        return set_error(ctx, CPDP_EINVAL, "tile %lld outside [0, %lld)", (long long)tile, (long long)tiles);
    ctx->tma_withheld_tile = tile;
    return CPDP_OK;
}

cpdp_status cpdp_reconcile_kernel(const cpdp_ctx* ctx, const char** name) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    if (name == nullptr) return set_error(nullptr, CPDP_EINVAL, "name is NULL");
    *name = ctx->reconcile_kernel;
    return CPDP_OK;
}

cpdp_status cpdp_wait_timeouts(cpdp_ctx* ctx, int64_t* count) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    if (count == nullptr) return set_error(ctx, CPDP_EINVAL, "count is NULL");
    if (ctx->device < 0) return set_error(ctx, CPDP_ESTATE, "state buffers not bound (call cpdp_bind first)");
    cpdp_status st = enter_device(ctx);
    if (st != CPDP_OK) return st;
    unsigned long long seen = 0, zero = 0;
    cudaError_t e = cudaDeviceSynchronize();
    if (e == cudaSuccess) e = cudaMemcpyFromSymbol(&seen, cpdp::tma_wait_timeouts, sizeof seen);
    if (e == cudaSuccess) e = cudaMemcpyToSymbol(cpdp::tma_wait_timeouts, &zero, sizeof zero);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "reading the wait-timeout count");
    *count = static_cast<int64_t>(seen);
    return CPDP_OK;
}

cpdp_status cpdp_set_optimizer_step(cpdp_ctx* ctx, int64_t step) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    if (step < 0) return set_error(ctx, CPDP_EINVAL, "optimizer step %lld < 0", (long long)step);
    ctx->opt_step = step;
    return CPDP_OK;
}

cpdp_status cpdp_get_optimizer_step(const cpdp_ctx* ctx, int64_t* step) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    if (step == nullptr) return set_error(nullptr, CPDP_EINVAL, "step is NULL");
    *step = ctx->opt_step;
    return CPDP_OK;
}

cpdp_status cpdp_get_counts(const cpdp_ctx* ctx, int64_t* grad_means, int64_t* param_means) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    if (grad_means != nullptr) *grad_means = ctx->grad_means;
    if (param_means != nullptr) *param_means = ctx->param_means;
    return CPDP_OK;
}

cpdp_status cpdp_step(cpdp_ctx* ctx, const void* grads, cpdp_dtype dtype, int64_t t, int64_t steps_per_epoch,
                      void* stream, int* did_sync) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    const int s = cpdp_is_sync_step(ctx, t, steps_per_epoch);
    if (s < 0)
        return set_error(ctx, CPDP_EINVAL, "step t=%lld outside [1, steps_per_epoch=%lld]", (long long)t,
                         (long long)steps_per_epoch);
    const cpdp_status st = s ? cpdp_reconcile(ctx, grads, dtype, stream) : cpdp_local_step(ctx, grads, dtype, stream);
    if (st == CPDP_OK && did_sync != nullptr) *did_sync = s;
    return st;
}

cpdp_status cpdp_set_lr(cpdp_ctx* ctx, float lr) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    if (!std::isfinite(lr) || !(lr > 0.f)) return set_error(ctx, CPDP_EINVAL, "lr=%g must be finite and > 0", (double)lr);
    ctx->lr = lr;
    return CPDP_OK;
}

cpdp_status cpdp_set_sync_period(cpdp_ctx* ctx, int K) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    if (K < 1) return set_error(ctx, CPDP_EINVAL, "K=%d must be >= 1", K);
    ctx->K = K;
    return CPDP_OK;
}

cpdp_status cpdp_set_schedule(cpdp_ctx* ctx, int64_t steps_per_epoch, int64_t total_epochs, int64_t warmup_epochs,
                              float base_lr, float min_lr) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    if (steps_per_epoch < 1 || total_epochs < 1 || warmup_epochs < 0 || warmup_epochs >= total_epochs)
        return set_error(ctx, CPDP_EINVAL, "schedule needs steps_per_epoch >= 1 and 0 <= warmup_epochs < total_epochs");
    if (total_epochs > (int64_t(1) << 40) / steps_per_epoch) return set_error(ctx, CPDP_EINVAL, "schedule too long");
    if (!finite_all({base_lr, min_lr}) || !(base_lr > 0.f) || min_lr < 0.f || min_lr > base_lr)
        return set_error(ctx, CPDP_EINVAL, "schedule needs finite 0 <= min_lr <= base_lr, base_lr > 0");
    ctx->has_schedule = true;
    ctx->sched_steps = steps_per_epoch;
    ctx->sched_epochs = total_epochs;
    ctx->sched_warmup = warmup_epochs;
    ctx->sched_base_lr = base_lr;
    ctx->sched_min_lr = min_lr;
    return CPDP_OK;
}

namespace {
bool in_schedule(const cpdp_ctx* c, int64_t epoch, int64_t t) {
    return c->has_schedule && epoch >= 0 && epoch < c->sched_epochs && t >= 1 && t <= c->sched_steps;
}
}  // namespace

float cpdp_scheduled_lr(const cpdp_ctx* ctx, int64_t epoch, int64_t t) {
    if (!usable(ctx) || !in_schedule(ctx, epoch, t)) return -1.0f;
    const int64_t s = epoch * ctx->sched_steps + (t - 1);
    const int64_t warm = ctx->sched_warmup * ctx->sched_steps;
    const int64_t total = ctx->sched_epochs * ctx->sched_steps;
    const double base = ctx->sched_base_lr, lo = ctx->sched_min_lr;
    if (s < warm) return static_cast<float>(base * static_cast<double>(s + 1) / static_cast<double>(warm));
    const double progress = static_cast<double>(s - warm) / static_cast<double>(total - warm);
    return static_cast<float>(lo + (base - lo) * 0.5 * (1.0 + std::cos(std::acos(-1.0) * progress)));
}

int cpdp_is_sync_step_at(const cpdp_ctx* ctx, int64_t epoch, int64_t t) {
    if (!usable(ctx) || !in_schedule(ctx, epoch, t)) return -1;
    if (epoch < ctx->sched_warmup) return 1;
    return cpdp_is_sync_step(ctx, t, ctx->sched_steps);
}

cpdp_status cpdp_step_at(cpdp_ctx* ctx, const void* grads, cpdp_dtype dtype, int64_t epoch, int64_t t, void* stream,
                         int* did_sync) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    if (!ctx->has_schedule) return set_error(ctx, CPDP_ESTATE, "no schedule set (call cpdp_set_schedule first)");
    if (!in_schedule(ctx, epoch, t))
        return set_error(ctx, CPDP_EINVAL, "step (epoch=%lld, t=%lld) outside the schedule", (long long)epoch,
                         (long long)t);
    cpdp_status st = enter_device(ctx);
    if (st != CPDP_OK) return st;
    if ((st = refuse_capture(ctx, static_cast<cudaStream_t>(stream),
                             "the learning-rate schedule advances every step")) != CPDP_OK)
        return st;
    const int s = cpdp_is_sync_step_at(ctx, epoch, t);
    const float prev_lr = ctx->lr;
    ctx->lr = cpdp_scheduled_lr(ctx, epoch, t);
    st = s ? cpdp_reconcile(ctx, grads, dtype, stream) : cpdp_local_step(ctx, grads, dtype, stream);
    if (st != CPDP_OK) {
        ctx->lr = prev_lr;
        return st;
    }
    if (did_sync != nullptr) *did_sync = s;
    return CPDP_OK;
}

}  // extern "C"

namespace {

// Copy one step's gradients from host memory into the next staging buffer on
// the copy stream, make `stream` wait for the copy, run `step` on the staged
// buffer, and mark the buffer free once `stream` has consumed it.
template <typename StepFn>
cpdp_status step_from_host(cpdp_ctx* ctx, const void* host_grads, cpdp_dtype dtype, void* stream, StepFn step) {
    if (ctx->copy_stream == nullptr) return set_error(ctx, CPDP_ESTATE, "no staging buffers (call cpdp_bind_staging first)");
    if (host_grads == nullptr) return set_error(ctx, CPDP_EINVAL, "host_grads is NULL");
    if (dtype != CPDP_F32 && dtype != CPDP_BF16) return set_error(ctx, CPDP_EINVAL, "unknown gradient dtype %d", (int)dtype);
    if (!aligned16(host_grads)) return set_error(ctx, CPDP_EALIGN, "host_grads is not 16-byte aligned");
    const size_t bytes = static_cast<size_t>(ctx->W) * static_cast<size_t>(ctx->N) *
                         (dtype == CPDP_F32 ? sizeof(float) : sizeof(uint16_t));
    if (bytes > ctx->staging_bytes) return set_error(ctx, CPDP_EINVAL, "staging buffers hold %zu bytes, step needs %zu",
                                                     ctx->staging_bytes, bytes);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cpdp_status st = enter_device(ctx);
    if (st != CPDP_OK) return st;
    if ((st = refuse_capture(ctx, s, "the staging buffers alternate per call")) != CPDP_OK) return st;
    if ((st = check_readable(ctx, host_grads, "host_grads")) != CPDP_OK) return st;
    const int k = static_cast<int>(ctx->staged & 1);
    cudaError_t e = cudaSuccess;
    if (ctx->staging_used[k]) e = cudaStreamWaitEvent(ctx->copy_stream, ctx->consumed[k], 0);
    if (e == cudaSuccess) e = cudaMemcpyAsync(ctx->staging[k], host_grads, bytes, cudaMemcpyDefault, ctx->copy_stream);
    if (e == cudaSuccess) e = cudaEventRecord(ctx->copied[k], ctx->copy_stream);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(s, ctx->copied[k], 0);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "staging copy");
    if ((st = step(ctx->staging[k])) != CPDP_OK) return st;
    if ((e = cudaEventRecord(ctx->consumed[k], s)) != cudaSuccess) return cuda_fail(ctx, e, "staging event");
    ctx->staging_used[k] = true;
    ++ctx->staged;
    return CPDP_OK;
}

void release_staging(cpdp_ctx* ctx) {
    for (int k = 0; k < 2; ++k) {
        if (ctx->copied[k] != nullptr) cudaEventDestroy(ctx->copied[k]);
        if (ctx->consumed[k] != nullptr) cudaEventDestroy(ctx->consumed[k]);
        ctx->copied[k] = ctx->consumed[k] = nullptr;
    }
    if (ctx->copy_stream != nullptr) cudaStreamDestroy(ctx->copy_stream);
    ctx->copy_stream = nullptr;
}

}  // namespace

extern "C" {

cpdp_status cpdp_bind_staging(cpdp_ctx* ctx, void* stage0, void* stage1, size_t bytes_each) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    if (ctx->params == nullptr) return set_error(ctx, CPDP_ESTATE, "state buffers not bound (call cpdp_bind first)");
    if (stage0 == nullptr || stage1 == nullptr) return set_error(ctx, CPDP_EINVAL, "a staging buffer is NULL");
    if (!aligned16(stage0) || !aligned16(stage1)) return set_error(ctx, CPDP_EALIGN, "staging buffers must be 16-byte aligned");
    if (bytes_each < static_cast<size_t>(ctx->W) * static_cast<size_t>(ctx->N) * sizeof(uint16_t))
        return set_error(ctx, CPDP_EINVAL, "staging buffers of %zu bytes cannot hold one step's gradients", bytes_each);
    if (overlaps(stage0, bytes_each, stage1, bytes_each) || overlaps_state(ctx, stage0, bytes_each) ||
        overlaps_state(ctx, stage1, bytes_each))
        return set_error(ctx, CPDP_EINVAL, "staging buffers overlap each other or the state");
    for (void* p : {stage0, stage1}) {
        cudaPointerAttributes at;
        const cudaError_t e = cudaPointerGetAttributes(&at, p);
        if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaPointerGetAttributes(staging)");
        if ((at.type != cudaMemoryTypeDevice && at.type != cudaMemoryTypeManaged) || at.device != ctx->device)
            return set_error(ctx, CPDP_EINVAL, "staging buffers must be device memory on the state's device");
    }
    cpdp_status st = enter_device(ctx);
    if (st != CPDP_OK) return st;
    if (ctx->copy_stream == nullptr) {
        cudaError_t e = cudaStreamCreateWithFlags(&ctx->copy_stream, cudaStreamNonBlocking);
        for (int k = 0; k < 2 && e == cudaSuccess; ++k) {
            e = cudaEventCreateWithFlags(&ctx->copied[k], cudaEventDisableTiming);
            if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ctx->consumed[k], cudaEventDisableTiming);
        }
        if (e != cudaSuccess) {
            release_staging(ctx);
            return cuda_fail(ctx, e, "copy stream / events");
        }
    } else {
        // rebinding: let copies into the old buffers finish first
        const cudaError_t e = cudaStreamSynchronize(ctx->copy_stream);
        if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaStreamSynchronize(copy stream)");
    }
    ctx->staging[0] = stage0;
    ctx->staging[1] = stage1;
    ctx->staging_bytes = bytes_each;
    ctx->staging_used[0] = ctx->staging_used[1] = false;
    ctx->staged = 0;
    return CPDP_OK;
}

cpdp_status cpdp_step_host(cpdp_ctx* ctx, const void* host_grads, cpdp_dtype dtype, int64_t t, int64_t steps_per_epoch,
                           void* stream, int* did_sync) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    if (cpdp_is_sync_step(ctx, t, steps_per_epoch) < 0)
        return set_error(ctx, CPDP_EINVAL, "step t=%lld outside [1, steps_per_epoch=%lld]", (long long)t,
                         (long long)steps_per_epoch);
    return step_from_host(ctx, host_grads, dtype, stream, [&](const void* staged) {
        return cpdp_step(ctx, staged, dtype, t, steps_per_epoch, stream, did_sync);
    });
}

cpdp_status cpdp_step_host_at(cpdp_ctx* ctx, const void* host_grads, cpdp_dtype dtype, int64_t epoch, int64_t t,
                              void* stream, int* did_sync) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    if (!ctx->has_schedule) return set_error(ctx, CPDP_ESTATE, "no schedule set (call cpdp_set_schedule first)");
    if (!in_schedule(ctx, epoch, t))
        return set_error(ctx, CPDP_EINVAL, "step (epoch=%lld, t=%lld) outside the schedule", (long long)epoch,
                         (long long)t);
    return step_from_host(ctx, host_grads, dtype, stream, [&](const void* staged) {
        return cpdp_step_at(ctx, staged, dtype, epoch, t, stream, did_sync);
    });
}

cpdp_status cpdp_destroy(cpdp_ctx* ctx) {
    if (ctx == nullptr) return CPDP_OK;
    {
        std::lock_guard<std::mutex> lock(g_live_mutex);
        auto& live = live_contexts();
        auto it = live.find(ctx);
        if (it == live.end()) return set_error(nullptr, CPDP_EINVAL, "cpdp_destroy: %p is not a live context", (void*)ctx);
        live.erase(it);
    }
    release_staging(ctx);
    ctx->magic = 0;
    delete ctx;
    return CPDP_OK;
}

cpdp_status cpdp_bad_index_count(cpdp_ctx* ctx, int64_t* count) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    if (count == nullptr) return set_error(ctx, CPDP_EINVAL, "count is NULL");
#ifdef CPDP_CHECKED
    if (ctx->device < 0) return set_error(ctx, CPDP_ESTATE, "state buffers not bound (call cpdp_bind first)");
    cpdp_status st = enter_device(ctx);
    if (st != CPDP_OK) return st;
    unsigned long long seen = 0, zero = 0;
    cudaError_t e = cudaDeviceSynchronize();
    if (e == cudaSuccess) e = cudaMemcpyFromSymbol(&seen, cpdp::bad_index_count, sizeof seen);
    if (e == cudaSuccess) e = cudaMemcpyToSymbol(cpdp::bad_index_count, &zero, sizeof zero);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "reading the bad-index count");
    *count = static_cast<int64_t>(seen);
#else
    *count = -1;  // a release build checks no index
#endif
    return CPDP_OK;
}

cpdp_status cpdp_floor_stream(const float* const* in, int n_in, const uint16_t* const* in_bf16, int n_in_bf16,
                              float* const* out, int n_out, int64_t n, unsigned grid, void* stream) {
    if (n_in < 0 || n_in > cpdp::kFloorMaxRows || n_in_bf16 < 0 || n_in_bf16 > cpdp::kFloorMaxRows ||
        n_in + n_in_bf16 < 1 || n_out < 0 || n_out > cpdp::kFloorMaxRows)
        return set_error(nullptr, CPDP_EINVAL,
                         "n_in=%d and n_in_bf16=%d in [0, %d] with at least one input row, and n_out=%d in [0, %d] "
                         "required",
                         n_in, n_in_bf16, cpdp::kFloorMaxRows, n_out, cpdp::kFloorMaxRows);
    if ((n_in > 0 && in == nullptr) || (n_in_bf16 > 0 && in_bf16 == nullptr) || (n_out > 0 && out == nullptr))
        return set_error(nullptr, CPDP_EINVAL, "row array is NULL");
    if (n < 4 || (n & 3) != 0) return set_error(nullptr, CPDP_EINVAL, "n=%lld must be a positive multiple of 4", (long long)n);
    cpdp::FloorRows rows{};
    rows.n_in = n_in;
    rows.n_in_bf16 = n_in_bf16;
    rows.n_out = n_out;
    for (int k = 0; k < n_in; ++k) {
        if (in[k] == nullptr || !aligned16(in[k])) return set_error(nullptr, CPDP_EALIGN, "input row %d NULL or not 16-byte aligned", k);
        rows.in[k] = in[k];
    }
    for (int k = 0; k < n_in_bf16; ++k) {
        if (in_bf16[k] == nullptr || reinterpret_cast<uintptr_t>(in_bf16[k]) % 8 != 0)
            return set_error(nullptr, CPDP_EALIGN, "bf16 input row %d NULL or not 8-byte aligned", k);
        rows.in_bf16[k] = reinterpret_cast<const cpdp::bf16_bits*>(in_bf16[k]);
    }
    for (int k = 0; k < n_out; ++k) {
        if (out[k] == nullptr || !aligned16(out[k])) return set_error(nullptr, CPDP_EALIGN, "output row %d NULL or not 16-byte aligned", k);
        rows.out[k] = out[k];
    }
    const int64_t nq = n >> 2;
    const unsigned g = grid != 0 ? grid : cpdp::grid_for(nq, cpdp::kThreads);
    const cudaError_t e = launch_shaped(true, cpdp::floor_stream_kernel, g, cpdp::kThreads, 0,
                                        static_cast<cudaStream_t>(stream), rows, nq);
    const cudaError_t e2 = e != cudaSuccess ? e : cudaGetLastError();
    if (e2 != cudaSuccess) return set_error(nullptr, CPDP_ECUDA, "floor_stream launch: %s", cudaGetErrorString(e2));
    return CPDP_OK;
}

cpdp_status cpdp_floor_empty(unsigned grid, void* stream) {
    const cudaError_t e = launch_shaped(true, cpdp::floor_empty_kernel, grid != 0 ? grid : 1u, cpdp::kThreads, 0,
                                        static_cast<cudaStream_t>(stream));
    const cudaError_t e2 = e != cudaSuccess ? e : cudaGetLastError();
    if (e2 != cudaSuccess) return set_error(nullptr, CPDP_ECUDA, "floor_empty launch: %s", cudaGetErrorString(e2));
    return CPDP_OK;
}

cpdp_status cpdp_floor_columns(float* params, float* mom, float* sq, const void* grads, cpdp_dtype grad_dtype,
                               float* anchor, float* slow_v, int W, int64_t N, int chunk_rows, int blocks_per_sm,
                               void* stream) {
    if (W < 1 || W > kMaxWorkers) return set_error(nullptr, CPDP_EINVAL, "W=%d must be in [1, %d]", W, kMaxWorkers);
    if (N < 4 || (N & 3) != 0) return set_error(nullptr, CPDP_EINVAL, "N=%lld must be a positive multiple of 4", (long long)N);
    if (grad_dtype != CPDP_F32 && grad_dtype != CPDP_BF16)
        return set_error(nullptr, CPDP_EINVAL, "unknown gradient dtype %d", (int)grad_dtype);
    if (!((chunk_rows == 2 && blocks_per_sm == 4) || (chunk_rows == 3 && blocks_per_sm == 3) ||
          (chunk_rows == 4 && blocks_per_sm == 2)))
        return set_error(nullptr, CPDP_EINVAL, "chunk_rows=%d, blocks_per_sm=%d: one of (2, 4), (3, 3), (4, 2) required",
                         chunk_rows, blocks_per_sm);
    const void* arrays[] = {params, mom, anchor, slow_v};
    for (const void* a : arrays)
        if (a == nullptr || !aligned16(a)) return set_error(nullptr, CPDP_EALIGN, "state array NULL or not 16-byte aligned");
    if (sq != nullptr && !aligned16(sq)) return set_error(nullptr, CPDP_EALIGN, "sq not 16-byte aligned");
    if (grads == nullptr || reinterpret_cast<uintptr_t>(grads) % (grad_dtype == CPDP_F32 ? 16 : 8) != 0)
        return set_error(nullptr, CPDP_EALIGN, "grads NULL or not aligned to a group of 4 elements");
    const cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int64_t nq = N >> 2;
    const cudaError_t e =
        grad_dtype == CPDP_F32
            ? launch_floor_columns_shape<float>(chunk_rows, blocks_per_sm, params, mom, sq, grads, anchor, slow_v, W, nq, s)
            : launch_floor_columns_shape<cpdp::bf16_bits>(chunk_rows, blocks_per_sm, params, mom, sq, grads, anchor,
                                                          slow_v, W, nq, s);
    const cudaError_t e2 = e != cudaSuccess ? e : cudaGetLastError();
    if (e2 != cudaSuccess) return set_error(nullptr, CPDP_ECUDA, "floor_columns launch: %s", cudaGetErrorString(e2));
    return CPDP_OK;
}

const char* cpdp_last_error(const cpdp_ctx* ctx) {
    if (ctx == nullptr) return t_error.c_str();
    if (!usable(ctx)) return "not a live context";
    return ctx->error.c_str();
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Host-fed step with a built-in staging area (cpdp_step_host_noalloc). The
// paper has no counterpart. It is cpdp_step_host for callers that cannot
// allocate device memory for cpdp_bind_staging: the staging area is a
// file-scope device array, reserved on every device where the library's
// device code is loaded and held until the process exits.
// ---------------------------------------------------------------------------
static __device__ __align__(256) unsigned char g_noalloc_staging[CPDP_NOALLOC_STAGING_BYTES];

namespace {

constexpr int kNoAllocMaxDevices = 64;
std::mutex g_noalloc_mutex;
void* g_noalloc_address[kNoAllocMaxDevices] = {};

// Device address of g_noalloc_staging on `device`, which must be the current
// device. In host code the array's name stands for the symbol only, not for
// device memory; the address comes from cudaGetSymbolAddress. It is looked up
// again on every call made outside stream capture (a host-side lookup that
// allocates nothing), so a device reset, which reloads the module and may move
// the array, is followed. A call under capture uses the address found by the
// last call on that device outside capture, or looks it up if there was none.
cpdp_status noalloc_staging(cpdp_ctx* ctx, int device, bool capturing, void** out) {
    if (device < 0 || device >= kNoAllocMaxDevices)
        return set_error(ctx, CPDP_EINVAL, "device %d is beyond the %d devices the built-in staging area serves", device,
                         kNoAllocMaxDevices);
    std::lock_guard<std::mutex> lock(g_noalloc_mutex);
    if (!capturing || g_noalloc_address[device] == nullptr) {
        void* ptr = nullptr;
        const cudaError_t e = cudaGetSymbolAddress((void**)&ptr, g_noalloc_staging);
        if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaGetSymbolAddress(built-in staging area)");
        g_noalloc_address[device] = ptr;
    }
    *out = g_noalloc_address[device];
    return CPDP_OK;
}

}  // namespace

extern "C" cpdp_status cpdp_step_host_noalloc(cpdp_ctx* ctx, const void* host_grads, cpdp_dtype dtype, int64_t t,
                                              int64_t steps_per_epoch, void* stream, int* did_sync) {
    if (!usable(ctx)) return set_error(nullptr, CPDP_EINVAL, "invalid context");
    if (ctx->params == nullptr) return set_error(ctx, CPDP_ESTATE, "state buffers not bound (call cpdp_bind first)");
    if (cpdp_is_sync_step(ctx, t, steps_per_epoch) < 0)
        return set_error(ctx, CPDP_EINVAL, "step t=%lld outside [1, steps_per_epoch=%lld]", (long long)t,
                         (long long)steps_per_epoch);
    if (host_grads == nullptr) return set_error(ctx, CPDP_EINVAL, "host_grads is NULL");
    if (dtype != CPDP_F32 && dtype != CPDP_BF16) return set_error(ctx, CPDP_EINVAL, "unknown gradient dtype %d", (int)dtype);
    if (!aligned16(host_grads)) return set_error(ctx, CPDP_EALIGN, "host_grads is not 16-byte aligned");
    const size_t bytes = static_cast<size_t>(ctx->W) * static_cast<size_t>(ctx->N) *
                         (dtype == CPDP_F32 ? sizeof(float) : sizeof(uint16_t));
    if (bytes > static_cast<size_t>(CPDP_NOALLOC_STAGING_BYTES))
        return set_error(ctx, CPDP_EINVAL,
                         "one step's gradients take %zu bytes (W*N*element size) but the built-in staging area "
                         "holds %zu; use cpdp_bind_staging with cpdp_step_host for this size",
                         bytes, static_cast<size_t>(CPDP_NOALLOC_STAGING_BYTES));
    cpdp_status st = enter_device(ctx);
    if (st != CPDP_OK) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    bool capturing = false;
    if ((st = capture_active(ctx, s, &capturing)) != CPDP_OK) return st;
    // every refusal cpdp_step would make comes before the copy, so a refused
    // call leaves nothing on the stream (nor in a graph being captured)
    if (capturing && ctx->optimizer == CPDP_OPT_ADAMW)
        return set_error(ctx, CPDP_ESTATE, "cannot be captured into a CUDA graph: %s",
                         "AdamW's bias correction depends on the step count");
    if ((st = check_readable(ctx, host_grads, "host_grads")) != CPDP_OK) return st;
    void* staging = nullptr;
    if ((st = noalloc_staging(ctx, ctx->device, capturing, &staging)) != CPDP_OK) return st;
    if ((st = check_grads(ctx, staging, dtype)) != CPDP_OK) return st;
    // copy on the caller's stream, so the step below reads it in stream order
    const cudaError_t e = cudaMemcpyAsync(staging, host_grads, bytes, cudaMemcpyDefault, s);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "copy into the built-in staging area");
    return cpdp_step(ctx, staging, dtype, t, steps_per_epoch, stream, did_sync);
}
