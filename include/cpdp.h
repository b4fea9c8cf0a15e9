/*
 * cpdp.h — C ABI of libcpdp, the GB300 (sm_103a) implementation of the
 * data-parallel hot path of CPDP (Controlled Periodic Data Parallelism with
 * SlowMo momentum).
 *
 * Model of the method (Algorithm 1 of the paper): W workers each hold a replica
 * theta_i of N parameters and a momentum buffer buf_i. At step t every worker
 * has a gradient g_i. If t is not a synchronization step (eq. 4) every worker
 * runs a local momentum-SGD update with its own gradient (eq. 5, Sec. 4.2).
 * Otherwise the reconcile runs: mean gradient (eq. 2), a synchronized
 * optimizer step on every worker through its own buffer (eq. 6), mean of the
 * replicas (eq. 7), the SlowMo update against the anchor theta_ref (eqs. 8-10)
 * and the write-back of the new model to every replica and to the anchor
 * (eqs. 11-12). Here the W workers are rows of buffers in one GPU's memory;
 * nothing crosses a GPU or a process.
 *
 * Memory layout (all caller-owned device memory, e.g. torch tensors):
 *   params  float32 [W][N]  replica of worker i at params + i*N
 *   mom     float32 [W][N]  per-worker momentum buffers (never averaged)
 *   anchor  float32 [N]     theta_ref
 *   slow_v  float32 [N]     SlowMo velocity v
 *   grads   float32 or bfloat16 [W][N], read only, row i = worker i
 * Row stride is exactly N elements. All pointers must be 16-byte aligned.
 * The fast vectorised kernels run when N is a multiple of 4; any other N runs
 * a scalar path with the same results.
 *
 * Optimizer step (the paper's implementation: PyTorch SGD, momentum 0.9,
 * weight decay 5e-4; Sec. 4.2, Table 3), per element:
 *   d = g + weight_decay * theta;  buf = momentum * buf + d;  theta -= lr * buf
 * SlowMo (eqs. 8-10), with alpha an outer step size the paper does not have
 * (alpha = 1 is the paper's update):
 *   v = beta * v + (theta_avg - theta_ref);  theta_new = theta_ref + alpha * v
 *
 * Errors: every call returns a cpdp_status. On failure cpdp_last_error() gives
 * a message. No call aborts, traps or throws across the ABI. Kernel launches
 * are asynchronous on the stream given; CUDA errors visible at launch time are
 * returned as CPDP_ECUDA, later device errors surface at the caller's next
 * synchronization. Thread safety: one context must not be used by two host
 * threads at once; distinct contexts are independent.
 *
 * CUDA graphs: cpdp_local_step, cpdp_reconcile and cpdp_step may be called on
 * a stream that is being captured, once each gradient buffer
 * has been used in one call outside capture (its memory type is checked then).
 * A captured launch keeps the arguments of the call that recorded it (the
 * learning rate, the method, the optimizer step), and replays do not advance
 * the context's host-side counters (cpdp_get_optimizer_step, cpdp_get_counts).
 * So replaying is exact for momentum SGD at a fixed learning rate, e.g. a
 * K-cycle captured once and replayed per synchronization period. Calls whose
 * replay would repeat a stale argument return CPDP_ESTATE under capture and
 * launch nothing: AdamW steps (bias correction depends on the step count),
 * cpdp_step_at (the learning-rate schedule advances per step), and the
 * host-fed steps (the staging buffers alternate per call).
 */
#ifndef CPDP_H
#define CPDP_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Opaque context, allocated and owned by the library (host memory only). */
typedef struct cpdp_ctx cpdp_ctx;

typedef enum {
    CPDP_OK = 0,
    CPDP_EINVAL = 1, /* an argument is out of range, null, or inconsistent */
    CPDP_EALIGN = 2, /* a pointer is not 16-byte aligned */
    CPDP_ECUDA = 3,  /* the CUDA runtime reported an error */
    CPDP_ESTATE = 4, /* call out of order (e.g. a step before cpdp_bind) */
    CPDP_ENOMEM = 5  /* host allocation failed */
} cpdp_status;

/* Element type of the gradient buffer. */
typedef enum {
    CPDP_F32 = 0,  /* IEEE float32 */
    CPDP_BF16 = 1  /* bfloat16 (upper 16 bits of a float32), widened exactly */
} cpdp_dtype;

/* Synchronization method (Sec. 5.4 compares the paper's method with two
 * baselines on the same optimizer):
 *   CPDP_METHOD_CPDP      the paper's method (the default): at a sync step,
 *                         gradient mean, synced step, parameter mean, SlowMo.
 *   CPDP_METHOD_LOCALSGD  at a sync step each worker steps with its own
 *                         gradient, then the parameters are averaged; no
 *                         gradient mean, no SlowMo (anchor and v unused).
 *   CPDP_METHOD_DDP       every step is a sync step (K = 1): gradient mean and
 *                         each worker's step with it; no parameter averaging. */
typedef enum {
    CPDP_METHOD_CPDP = 0,
    CPDP_METHOD_LOCALSGD = 1,
    CPDP_METHOD_DDP = 2
} cpdp_method;

/* Each worker's optimizer. CPDP_OPT_SGD (the default): momentum SGD with
 * coupled weight decay (the paper's ResNet-50 runs). CPDP_OPT_ADAMW: AdamW
 * with decoupled weight decay and bias-corrected moments (the paper's ViT-S
 * runs, Sec. 5.2, Table 3), enabled by cpdp_set_adamw. */
typedef enum {
    CPDP_OPT_SGD = 0,
    CPDP_OPT_ADAMW = 1
} cpdp_optimizer;

/*
 * cpdp_create — validate the problem and hyperparameters, allocate a context.
 * Host-only: touches no GPU, so it can be called on a machine without one.
 *   out            receives the new context (set to NULL on failure)
 *   W              number of simulated workers, 1 <= W <= 4096 (the paper's N)
 *   N              parameters per replica, N >= 1 (the paper's d), with
 *                  W * N <= 2^40
 *   tensor_offsets num_tensors+1 prefix offsets of the model's tensors in the
 *                  flat parameter vector: [0] = 0, strictly increasing,
 *                  [num_tensors] = N. Copied; the caller keeps ownership. The
 *                  update is elementwise, so the table does not change the
 *                  result; it records the model's layout. May be NULL when
 *                  num_tensors == 0, meaning one tensor of N elements.
 *   lr             learning rate eta > 0 (Sec. 3.1 boundary conditions)
 *   momentum       SGD momentum mu >= 0
 *   weight_decay   coupled L2 weight decay lambda >= 0
 *   K              synchronization period, K >= 1 (eq. 4; K = 1 is DDP)
 *   slowmo_beta    SlowMo coefficient beta in [0, 1) (Sec. 3.1, Sec. 3.3)
 *   slowmo_alpha   outer step size alpha > 0 (1 = the paper's eq. 10)
 * All floating-point arguments must be finite.
 */
cpdp_status cpdp_create(cpdp_ctx **out, int W, int64_t N,
                        const int64_t *tensor_offsets, int num_tensors,
                        float lr, float momentum, float weight_decay, int K,
                        float slowmo_beta, float slowmo_alpha);

/*
 * cpdp_bind — attach the caller's state buffers (layout above). The library
 * keeps non-owning pointers; the caller keeps the memory alive and unmoved
 * until cpdp_destroy or the next cpdp_bind. Checks: non-null (EINVAL), 16-byte
 * aligned (EALIGN), device or managed memory on one device (EINVAL/ECUDA), and
 * no two of the four ranges overlapping (EINVAL). Makes that device current.
 */
cpdp_status cpdp_bind(cpdp_ctx *ctx, float *params, float *mom, float *anchor,
                      float *slow_v);

/*
 * cpdp_init_params — Algorithm 1 initialisation: every replica and the anchor
 * take theta0, the momentum buffers and the SlowMo velocity become 0.
 *   theta0  float32 [N] device or page-locked host memory, 16-byte aligned,
 *           not overlapping the state (pageable host memory: CPDP_EINVAL)
 *   stream  a cudaStream_t (NULL = legacy default stream)
 */
cpdp_status cpdp_init_params(cpdp_ctx *ctx, const float *theta0, void *stream);

/*
 * cpdp_local_step — local update phase (s_t = 0; eq. 5 with the momentum-SGD
 * step of Sec. 4.2, or AdamW after cpdp_set_adamw): every worker i updates
 * theta_i and its optimizer state with its own gradient row g_i. One kernel
 * launch over all W replicas.
 *   grads  [W][N] of `dtype`, device memory or page-locked host memory, 16-byte
 *          aligned; read only
 */
cpdp_status cpdp_local_step(cpdp_ctx *ctx, const void *grads, cpdp_dtype dtype,
                            void *stream);

/*
 * cpdp_reconcile — synchronization phase (s_t = 1; eqs. 2, 6-12 and the sync
 * branch of Algorithm 1), fused into one kernel launch: per parameter it reads
 * the W gradients, forms their mean, applies each worker's momentum step with
 * that mean, averages the W stepped replicas, applies SlowMo against the
 * anchor, and writes the same new value to all W replicas, the anchor and v.
 * Momentum buffers are updated per worker and are not averaged (Sec. 4.2)
 * unless cpdp_set_state_reconcile is on. cpdp_set_method selects the
 * baselines' sync steps instead (LocalSGD, DDP) on the same launch. Under CPDP
 * and LocalSGD all W replica rows are bit-identical after the call.
 */
cpdp_status cpdp_reconcile(cpdp_ctx *ctx, const void *grads, cpdp_dtype dtype,
                           void *stream);

/*
 * cpdp_is_sync_step — the synchronization indicator s_t of eq. 4 with the
 * epoch-end rule of Sec. 3.1: for 1-based step t in an epoch of
 * steps_per_epoch mini-batches, returns 1 iff t mod K == 0 or
 * t == steps_per_epoch (always 1 under CPDP_METHOD_DDP), 0 if not, and -1 on
 * invalid arguments (ctx NULL, t < 1, or t > steps_per_epoch). Host-only.
 */
int cpdp_is_sync_step(const cpdp_ctx *ctx, int64_t t, int64_t steps_per_epoch);

/*
 * cpdp_step — one mini-batch step of Algorithm 1: runs cpdp_reconcile if
 * cpdp_is_sync_step(ctx, t, steps_per_epoch) is 1, else cpdp_local_step.
 * If did_sync is not NULL it receives 1 or 0 accordingly.
 */
cpdp_status cpdp_step(cpdp_ctx *ctx, const void *grads, cpdp_dtype dtype,
                      int64_t t, int64_t steps_per_epoch, void *stream,
                      int *did_sync);

/*
 * cpdp_set_lr — change the learning rate for subsequent steps (for a schedule
 * driven by the caller; cpdp_step_at below drives the paper's own).
 * lr must be finite and > 0. Host-only.
 */
cpdp_status cpdp_set_lr(cpdp_ctx *ctx, float lr);

/*
 * cpdp_set_method — select the synchronization method (cpdp_method above) for
 * subsequent cpdp_reconcile / cpdp_step calls; cpdp_local_step is the same in
 * every method. Host-only.
 */
cpdp_status cpdp_set_method(cpdp_ctx *ctx, cpdp_method method);

/*
 * cpdp_set_adamw — switch every worker's optimizer to AdamW (the optimizer of
 * the paper's ViT-S runs; Sec. 5.2, Table 3) and bind its second-moment
 * buffer. Call after cpdp_bind. Per element, with t the 1-based optimizer step
 * count, lr the current learning rate and wd the weight_decay given to
 * cpdp_create (decoupled; momentum is unused):
 *   theta *= 1 - lr * wd
 *   m = beta1 * m + (1 - beta1) * g;   s = beta2 * s + (1 - beta2) * g * g
 *   theta -= (lr / (1 - beta1^t)) * m / (sqrt(s) / sqrt(1 - beta2^t) + eps)
 * evaluated in float32 with the factors of t formed in double on the host (the
 * division by sqrt(1 - beta2^t) is a multiplication by its reciprocal) and a
 * fast division for m / (...) accurate to a few ulps. The first moments m live in the `mom` buffer given to cpdp_bind; the second
 * moments s in exp_avg_sq (float32 [W][N], caller-owned device memory, 16-byte
 * aligned, on the state's device, not overlapping the other buffers). Both
 * stay per worker (Sec. 4.2). The step count is shared by all workers, starts
 * at 0 here and at cpdp_init_params (which also zeroes exp_avg_sq), and
 * advances by one on every cpdp_local_step / cpdp_reconcile.
 *   beta1, beta2 in [0, 1); eps finite and >= 0.
 */
cpdp_status cpdp_set_adamw(cpdp_ctx *ctx, float beta1, float beta2, float eps, float *exp_avg_sq);

/*
 * cpdp_set_state_reconcile — the optimizer-state reconciliation variant that
 * the paper names but does not use (Sec. 4.2, Sec. 6). With enable = 1, every
 * CPDP or LocalSGD synchronization step also replaces each worker's momentum
 * buffer (AdamW: both moments) by the mean over the workers of the post-step
 * states, so all workers leave the step with identical optimizer state. DDP is
 * unaffected (its states are identical by construction). enable = 0 (the
 * default) keeps the paper's behaviour: states stay per worker. Host-only.
 */
cpdp_status cpdp_set_state_reconcile(cpdp_ctx *ctx, int enable);

/*
 * cpdp_set_pdl — programmatic dependent launch for the context's kernels
 * (enable = 1, the default): each launch may begin while the previous grid on
 * the stream drains, which hides the gap between back-to-back kernels (about
 * 3 us each on GB300: +0.5 % per K-cycle at the ResNet-50 shape, +14 % at
 * N = 2^20, W = 8). Every kernel waits for the previous grid's completion
 * before touching memory, so results are bit-identical with enable = 0, which
 * launches with plain stream order. A CUDA event or other non-kernel work
 * between two launches restores plain stream order there. Host-only.
 */
cpdp_status cpdp_set_pdl(cpdp_ctx *ctx, int enable);

/*
 * cpdp_set_reconcile_staging — how cpdp_reconcile moves its rows (the
 * reconcile of Sec. 3.2-3.3: eqs. 2 and 7 read W rows per column). stages = 0
 * (the default): every thread loads its columns of the W rows straight from
 * global memory into registers. stages = 2..8: the rows pass through shared
 * memory instead: a producer warp copies tiles of 512 columns of every row
 * (W gradient, W parameter and W momentum rows, theta_ref, v) with bulk
 * copies (TMA, cp.async.bulk) into a ring of `stages` slots, consumer warps
 * reconcile a slot in place, and the updated rows go back with bulk stores.
 * The result is bit-identical to stages = 0; it is kept as the measured
 * alternative (slower on GB300: the staging adds a shared-memory pass and a
 * bulk-copy issue per 2 KB row segment without saving DRAM traffic).
 * Covers the CPDP method with momentum SGD, float32 gradients and no state
 * reconciliation; cpdp_reconcile returns CPDP_ESTATE for other settings while
 * it is on. Needs the state bound (else CPDP_ESTATE), W <= 16 and N a
 * multiple of 4, and `stages` slots of (3W + 2) * 2 KB within a block's
 * shared memory (else CPDP_EINVAL), and cpdp_set_reconcile_shuffle off (else
 * CPDP_ESTATE). Sets the kernel's shared-memory limit on the context's device;
 * launches nothing.
 */
cpdp_status cpdp_set_reconcile_staging(cpdp_ctx *ctx, int stages);

/*
 * cpdp_set_reconcile_shuffle — enable = 1: cpdp_reconcile splits the W worker
 * rows across the lanes of a warp instead of keeping a column's W rows in one
 * thread (the reconcile of Sec. 3.2-3.3; the W-way means of eqs. 2 and 7). A
 * warp covers 8 groups of 4 columns (128 bytes of a row); each lane takes one
 * group and every fourth row, sums its rows, and the four partial sums of a
 * group are added with two warp shuffles (__shfl_xor_sync). The replicas stay
 * bit-identical; from W = 4 on the sums run in a different order, so results
 * match enable = 0 to rounding (within the tests' 1e-5), not bit for bit. Kept
 * as the measured alternative to the register sums of enable = 0 (the
 * default): with 128-byte row segments per warp it reads each row in shorter
 * pieces. Covers the CPDP method with momentum SGD, float32 gradients and no
 * state reconciliation; cpdp_reconcile returns CPDP_ESTATE for other settings
 * while it is on. N must be a multiple of 4 (else CPDP_EINVAL); CPDP_ESTATE
 * while cpdp_set_reconcile_staging is on (and cpdp_set_reconcile_staging
 * returns CPDP_ESTATE while this is on). Host-only.
 */
cpdp_status cpdp_set_reconcile_shuffle(cpdp_ctx *ctx, int enable);

/*
 * cpdp_reconcile_kernel — sets *name to the name of the kernel that the last
 * reconcile on ctx launched (cpdp_reconcile, or a reconcile step of
 * cpdp_step, cpdp_step_at or the host-fed calls): "reconcile_vec4_kernel",
 * "reconcile_onepass_kernel", "reconcile_scalar_kernel",
 * "reconcile_tma_kernel" or "reconcile_shuffle_kernel"; "" before the first
 * one. The launch shape is chosen per worker count, method, optimizer, state
 * reconciliation and gradient type, so this tells a caller (a profile, a
 * benchmark) which kernel ran. The string is static: never freed, valid for
 * the life of the library. Host-only; an invalid ctx or a NULL name returns
 * CPDP_EINVAL and leaves *name unchanged.
 */
cpdp_status cpdp_reconcile_kernel(const cpdp_ctx *ctx, const char **name);

/*
 * cpdp_wait_timeouts — the number of bounded waits in the library's kernels
 * that ran out since the previous call (on any context of ctx's device), then
 * resets it. The staged reconcile's producer and consumer warps wait on
 * shared-memory barriers; a wait that has not ended after 2 s gives up, is
 * counted here, and its block stops working and returns once its copies have
 * landed (its results are then incomplete). 0 in correct operation. Waits
 * for all work on ctx's device (cudaDeviceSynchronize); needs the state
 * bound, else CPDP_ESTATE.
 */
cpdp_status cpdp_wait_timeouts(cpdp_ctx *ctx, int64_t *count);

/*
 * cpdp_withhold_staged_tile — a test of the staged reconcile's bounded waits
 * (the paper has no counterpart). In the next cpdp_reconcile on ctx (staging
 * on), the load warp leaves out the loads of column tile `tile` (512 columns,
 * 0 <= tile < ceil(N / 512)). The warps that wait for that tile give up after
 * 2 s each (about 4 s in all), count the waits in cpdp_wait_timeouts, and the
 * launch ends; the tile's columns are left part-updated, the rest reconciled.
 * Applies to one launch, then clears. CPDP_ESTATE when staging is off,
 * CPDP_EINVAL for a tile outside the range. Host-only.
 */
cpdp_status cpdp_withhold_staged_tile(cpdp_ctx *ctx, int64_t tile);

/*
 * cpdp_set_optimizer_step / cpdp_get_optimizer_step — the shared optimizer
 * step count (AdamW's bias correction uses it), e.g. to resume from a
 * checkpoint. step >= 0. Host-only.
 */
cpdp_status cpdp_set_optimizer_step(cpdp_ctx *ctx, int64_t step);
cpdp_status cpdp_get_optimizer_step(const cpdp_ctx *ctx, int64_t *step);

/*
 * cpdp_get_counts — how many gradient means and parameter means the context
 * has launched since creation: the in-memory counterparts of the paper's
 * gradient and parameter AllReduces (Table 2: per post-warmup epoch of T steps,
 * DDP T and 0, LocalSGD 0 and ceil(T/K), CPDP ceil(T/K) and ceil(T/K)).
 * Either pointer may be NULL. Host-only.
 */
cpdp_status cpdp_get_counts(const cpdp_ctx *ctx, int64_t *grad_means, int64_t *param_means);

/*
 * cpdp_set_sync_period — change the synchronization period K (K >= 1) for
 * subsequent steps, e.g. K = 1 during warmup epochs and the configured K
 * afterwards (Sec. 4.3, Sec. 5.4). Host-only.
 */
cpdp_status cpdp_set_sync_period(cpdp_ctx *ctx, int K);

/*
 * Training-protocol schedule (Sec. 4.3: cosine annealing with linear warmup;
 * warmup epochs run with K = 1). The paper prints no formula; this library
 * uses, for 0-based global step s = epoch * steps_per_epoch + (t - 1),
 * Sw = warmup_epochs * steps_per_epoch and S = total_epochs * steps_per_epoch:
 *   s <  Sw: lr = base_lr * (s + 1) / Sw                         (linear warmup)
 *   s >= Sw: lr = min_lr + (base_lr - min_lr) * (1 + cos(pi * (s - Sw) / (S - Sw))) / 2
 * computed in double precision and rounded to float.
 *
 * cpdp_set_schedule — enable the schedule. steps_per_epoch >= 1,
 *   total_epochs >= 1, 0 <= warmup_epochs < total_epochs, base_lr finite > 0,
 *   0 <= min_lr <= base_lr. Host-only.
 * cpdp_scheduled_lr — the schedule's learning rate for (0-based epoch, 1-based
 *   t); returns -1.0f if no schedule is set or the step is outside it.
 * cpdp_is_sync_step_at — 1 if step (epoch, t) synchronizes: every step of a
 *   warmup epoch, otherwise cpdp_is_sync_step's rule; 0 if not; -1 on invalid
 *   arguments or no schedule.
 * cpdp_step_at — one step of the protocol: sets the learning rate to
 *   cpdp_scheduled_lr(epoch, t), then runs cpdp_reconcile if
 *   cpdp_is_sync_step_at(epoch, t) is 1, else cpdp_local_step. The learning
 *   rate stays set afterwards (as by cpdp_set_lr).
 */
cpdp_status cpdp_set_schedule(cpdp_ctx *ctx, int64_t steps_per_epoch, int64_t total_epochs,
                              int64_t warmup_epochs, float base_lr, float min_lr);
float cpdp_scheduled_lr(const cpdp_ctx *ctx, int64_t epoch, int64_t t);
int cpdp_is_sync_step_at(const cpdp_ctx *ctx, int64_t epoch, int64_t t);
cpdp_status cpdp_step_at(cpdp_ctx *ctx, const void *grads, cpdp_dtype dtype, int64_t epoch,
                         int64_t t, void *stream, int *did_sync);

/*
 * Gradients that arrive in host memory (the end-to-end setting).
 *
 * cpdp_bind_staging — attach two caller-owned device staging buffers of
 *   bytes_each bytes each (>= W*N*sizeof(gradient element); device memory on
 *   the state's device, 16-byte aligned, not overlapping each other or the
 *   state). On the first call the library creates its own copy stream and four
 *   events, released by cpdp_destroy. Rebinding waits for copies in flight.
 * cpdp_step_host / cpdp_step_host_at — cpdp_step / cpdp_step_at on gradients
 *   read from `host_grads` ([W][N] of `dtype`, page-locked host memory; device
 *   memory is accepted too; pageable host memory is CPDP_EINVAL). The copy is
 *   issued on the library's copy stream into the staging buffers in turn; the
 *   step on `stream` waits for its copy (a stream-ordered event, no host
 *   synchronisation), and a staging buffer is refilled only after the step
 *   that read it. So the copy of step i+1 overlaps the kernels of step i. The
 *   caller must keep host_grads unchanged until the step that reads it has run
 *   (e.g. until an event recorded on `stream` after the call completes).
 */
cpdp_status cpdp_bind_staging(cpdp_ctx *ctx, void *stage0, void *stage1, size_t bytes_each);
cpdp_status cpdp_step_host(cpdp_ctx *ctx, const void *host_grads, cpdp_dtype dtype, int64_t t,
                           int64_t steps_per_epoch, void *stream, int *did_sync);
cpdp_status cpdp_step_host_at(cpdp_ctx *ctx, const void *host_grads, cpdp_dtype dtype, int64_t epoch,
                              int64_t t, void *stream, int *did_sync);

/*
 * cpdp_step_host_noalloc — cpdp_step_host without caller-provided staging
 * buffers. The paper has no counterpart: this is for callers that cannot
 * allocate device memory of their own. Examples are a process whose device
 * memory is already handed out by another allocator (a framework's caching
 * pool, a fixed-size arena), and a step loop that must not call cudaMalloc,
 * which can synchronize the device and stall work on other streams.
 * The caller still provides the state (cpdp_bind) and the gradients.
 *
 * The step's gradients, W*N elements of `dtype` from `host_grads` (page-locked
 * host memory or device memory; pageable host memory is CPDP_EINVAL), are
 * copied on `stream` into a staging area built into the library. Then
 * cpdp_step runs on them on the same stream. The area holds at most
 * CPDP_NOALLOC_STAGING_BYTES (64 MiB, e.g. W*N up to 16,777,216 float32 or
 * 33,554,432 bfloat16 elements); a larger step returns CPDP_EINVAL, names
 * the limit, and launches nothing. Every device where the library's device
 * code is loaded holds this area until the process exits. The entry point
 * itself calls no cudaMalloc, cudaFree or other allocating routine.
 *
 * Each call made outside stream capture looks up the area's device address
 * (cudaGetSymbolAddress, which allocates nothing), so the address stays right
 * after a device reset (cudaDeviceReset reloads the library's device code, and
 * the area may move). A call under capture reuses the address the last call on
 * that device found outside capture; make the first call on each device before
 * any stream capture. Every check that would refuse the step (arguments,
 * sizes, and, for AdamW, stream capture: CPDP_ESTATE) is made before the copy
 * is queued, so a refused call queues nothing on `stream`.
 * There is one area per device, shared by every call and
 * every context on that device: calls whose work can overlap on the GPU
 * (different streams, or contexts with no ordering between their streams)
 * race on it. Calls on one stream are ordered. The area keeps the last
 * call's gradients; each call overwrites the bytes it reads before reading
 * them, so nothing needs clearing. The caller must keep host_grads unchanged
 * until the copy has run (e.g. until an event recorded on `stream` after the
 * call completes).
 */
#define CPDP_NOALLOC_STAGING_BYTES (64u << 20)
cpdp_status cpdp_step_host_noalloc(cpdp_ctx *ctx, const void *host_grads, cpdp_dtype dtype, int64_t t,
                                   int64_t steps_per_epoch, void *stream, int *did_sync);

/*
 * cpdp_bad_index_count — a debugging aid for the library's own kernels. In the
 * debug build compiled with -DCPDP_CHECKED (libcpdp_checked.so), every kernel
 * checks each global-memory index against the extent of the buffer it
 * addresses; an index outside it is counted and replaced by 0, so the access
 * stays in bounds and nothing traps. This call waits for all work on ctx's
 * device (cudaDeviceSynchronize), stores the count since the previous call in
 * *count and resets it; it needs the state bound (cpdp_bind), else
 * CPDP_ESTATE. A release build stores -1 and waits for nothing.
 */
cpdp_status cpdp_bad_index_count(cpdp_ctx *ctx, int64_t *count);

/*
 * cpdp_destroy — free the context (and the copy stream and events of
 * cpdp_bind_staging, once their work completes). NULL is accepted (returns
 * CPDP_OK). A pointer that is not a live context (e.g. destroyed twice)
 * returns CPDP_EINVAL and is not touched. Never frees the caller's buffers.
 */
cpdp_status cpdp_destroy(cpdp_ctx *ctx);

/*
 * Measurement aids (the paper has no counterpart): the floors that a launch
 * of the hot path is compared with: where its data is small enough that
 * launch latency and ramp-up decide its time (e.g. W = 2, N = 2^20), and at
 * any size the same bytes moved in the same order with no arithmetic.
 *
 * cpdp_floor_stream — one launch of a plain streaming kernel on `stream`: for
 *   every group of 4 columns j < n, the sum of the n_in_bf16 bfloat16 rows
 *   in_bf16[k][j] (widened to float) and the n_in float32 rows in[k][j] is
 *   written to each of the n_out float32 rows out[k][j]. Given the rows a
 *   cpdp_local_step or cpdp_reconcile launch touches (outputs among the
 *   inputs, in place; bf16 gradients as bf16 rows), it moves the same bytes
 *   with the same read:write mix with no optimizer arithmetic, and for a
 *   reconcile walks the rows column by column as the reconcile does. Rows:
 *   device pointers, n elements each, n a positive multiple of 4; float32
 *   rows 16-byte aligned, bf16 rows 8-byte aligned; 0 <= n_in, n_in_bf16 <=
 *   128 with at least one input row, 0 <= n_out <= 128; in (in_bf16, out) may
 *   be NULL where n_in (n_in_bf16, n_out) is 0. grid = 0: one group of 4
 *   columns per thread (256 threads per block);
 *   else that many blocks, each thread looping over the columns. Bad
 *   arguments: CPDP_EINVAL / CPDP_EALIGN, nothing launched. Programmatic
 *   dependent launch on, like the context's kernels.
 *   The rows must be device memory of the current device: the call checks
 *   their alignment but not where they point, since a check of every row
 *   would cost more host time than the launch it is there to time.
 * cpdp_floor_empty — one launch of `grid` (0: 1) blocks of an empty kernel on
 *   `stream`: the cost of a launch.
 * Errors are reported by cpdp_last_error(NULL).
 */
cpdp_status cpdp_floor_stream(const float *const *in, int n_in, const uint16_t *const *in_bf16, int n_in_bf16,
                              float *const *out, int n_out, int64_t n, unsigned grid, void *stream);
cpdp_status cpdp_floor_empty(unsigned grid, void *stream);

/*
 * cpdp_floor_columns — one launch on `stream` of a kernel that walks a CPDP
 * reconcile's rows the way the reconcile does (a thread owns a group of 4
 * columns and visits rows 0 .. W-1 in chunks of chunk_rows, then theta_ref and
 * v) and reads and writes each row in place with no sum over the rows and no
 * dependency between them: per row params += g, mom += g and, where sq is not
 * NULL, sq += g; then anchor += slow_v. It moves a reconcile's algorithmic
 * bytes in the reconcile's order without its arithmetic: the rate of that
 * access pattern on its own. Arrays: device pointers laid out as for
 * cpdp_bind ([W][N] float32 rows; anchor and slow_v [N]), 16-byte aligned;
 * grads [W][N] of grad_dtype, aligned to a group of 4 elements; sq may be
 * NULL. 1 <= W <= 4096; N a positive multiple of 4; (chunk_rows,
 * blocks_per_sm) one of (2, 4), (3, 3), (4, 2) (the resident blocks per SM the
 * kernel is compiled for; none of the three spills). Bad arguments: CPDP_EINVAL / CPDP_EALIGN, nothing
 * launched. Overwrites the arrays it is given. Programmatic dependent launch
 * on. Errors are reported by cpdp_last_error(NULL).
 */
cpdp_status cpdp_floor_columns(float *params, float *mom, float *sq, const void *grads, cpdp_dtype grad_dtype,
                               float *anchor, float *slow_v, int W, int64_t N, int chunk_rows, int blocks_per_sm,
                               void *stream);

/*
 * cpdp_last_error — message of the last failed call on ctx, or, for ctx ==
 * NULL, of the last failed call on this host thread that had no context
 * (e.g. cpdp_create). Empty string if none. The pointer stays valid until the
 * next call on the same context / thread.
 */
const char *cpdp_last_error(const cpdp_ctx *ctx);

#ifdef __cplusplus
}
#endif

#endif /* CPDP_H */
