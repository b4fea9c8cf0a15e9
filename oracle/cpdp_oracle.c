/*
 * fp64 CPU oracle for the data-parallel hot path of CPDP (Controlled Periodic
 * Data Parallelism with SlowMo momentum).
 *
 * TEST INFRASTRUCTURE. Only the test suite, the smoke check and the benchmark's
 * CPU-baseline / reference arm load this library. The CUDA product path never
 * links, loads or calls it, and the two share no code, header or constant.
 *
 * What it computes: Algorithm 1 of the paper (CPDP with SlowMo outer momentum),
 * step by step and in the paper's order, on W workers' replicas held in one
 * address space. The optimizer update of both the local branch (eq. 5) and the
 * synchronized branch (eq. 6) is the one the paper's implementation runs
 * (Sec. 4.2: optimizer.step(); Table 3 / Sec. 5.2: SGD with momentum 0.9 and
 * weight decay 5e-4), i.e. PyTorch's SGD with coupled L2 weight decay, no
 * dampening and no Nesterov term:
 *     d = g + wd * theta;   buf = mu * buf + d;   theta = theta - lr * buf.
 * With mu = 0 and wd = 0 this is eq. 5 / eq. 6 literally.
 *
 * Layout: W rows of N doubles, row-major; worker i, parameter j at [i*N + j].
 * All arithmetic is double precision, single-threaded, plain loops; build with
 * -O2 -ffp-contract=off so that no multiply-add is fused.
 *
 * Pins: every function here is checked against hand-derived worked examples,
 * closed forms and library routines by the CPU test suite (tests/golden and
 * tests/oracle_pins.py); none is "parity unpinned".
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>

/* Algorithm 1, initialisation: every worker starts from the initial
 * parameters theta0, the SlowMo velocity v starts at 0 and the reference
 * (anchor) model theta_ref at theta0. Each worker's optimizer starts with an
 * empty momentum buffer; for the SGD update above an empty buffer behaves as a
 * buffer of zeros (its first step stores d, and mu * 0 + d = d). */
void oracle_init(int W, int64_t N, const double *theta0,
                 double *theta, double *buf, double *theta_ref, double *v)
{
    for (int i = 0; i < W; ++i) {
        for (int64_t j = 0; j < N; ++j) {
            theta[(int64_t)i * N + j] = theta0[j];
            buf[(int64_t)i * N + j] = 0.0;
        }
    }
    for (int64_t j = 0; j < N; ++j) {
        theta_ref[j] = theta0[j];
        v[j] = 0.0;
    }
}

/* One optimizer.step() of one worker: momentum SGD with coupled weight decay
 * (Sec. 4.2, Table 3), applied to the N parameters of that worker with the
 * gradient `grad`. */
static void sgd_momentum_update(int64_t N, double lr, double mu, double wd,
                                const double *grad, double *theta, double *buf)
{
    for (int64_t j = 0; j < N; ++j) {
        double d = grad[j] + wd * theta[j];
        buf[j] = mu * buf[j] + d;
        theta[j] = theta[j] - lr * buf[j];
    }
}

/* Local update phase (s_t = 0; eq. 5 and the local branch of Algorithm 1):
 * every worker i steps with its own gradient g_i. No data crosses workers. */
void oracle_local_step(int W, int64_t N, double lr, double mu, double wd,
                       const double *g, double *theta, double *buf)
{
    for (int i = 0; i < W; ++i) {
        sgd_momentum_update(N, lr, mu, wd, g + (int64_t)i * N,
                            theta + (int64_t)i * N, buf + (int64_t)i * N);
    }
}

/* Synchronization phase (s_t = 1; Sec. 3.2 stages one and two, Sec. 3.3, and
 * the sync branch of Algorithm 1), in the paper's order:
 *   1. gbar = (1/W) sum_i g_i                                  (eq. 2)
 *   2. every worker steps with gbar through its own optimizer  (eq. 6; the
 *      momentum buffers stay per worker, Sec. 4.2)
 *   3. theta_avg = (1/W) sum_i theta_i                         (eq. 7)
 *   4. delta = theta_avg - theta_ref; v = beta * v + delta;
 *      theta_new = theta_ref + alpha * v                       (eqs. 8-10)
 *   5. theta_i = theta_new for every worker; theta_ref = theta_new
 *                                                              (eqs. 11-12)
 * alpha is an outer step size that the paper does not have; alpha = 1 gives
 * eqs. 8-10 exactly. The momentum buffers are not averaged or reset.
 * Returns 0, or -1 if the temporaries could not be allocated. */
int oracle_reconcile(int W, int64_t N, double lr, double mu, double wd,
                     double beta, double alpha, const double *g,
                     double *theta, double *buf, double *theta_ref, double *v)
{
    double *gbar = (double *)malloc((size_t)N * sizeof(double));
    double *theta_avg = (double *)malloc((size_t)N * sizeof(double));
    double *theta_new = (double *)malloc((size_t)N * sizeof(double));
    if (gbar == NULL || theta_avg == NULL || theta_new == NULL) {
        free(gbar);
        free(theta_avg);
        free(theta_new);
        return -1;
    }

    /* 1. gradient mean over workers */
    for (int64_t j = 0; j < N; ++j) {
        double s = 0.0;
        for (int i = 0; i < W; ++i) s += g[(int64_t)i * N + j];
        gbar[j] = s / (double)W;
    }

    /* 2. synchronized optimizer step on every worker */
    for (int i = 0; i < W; ++i) {
        sgd_momentum_update(N, lr, mu, wd, gbar,
                            theta + (int64_t)i * N, buf + (int64_t)i * N);
    }

    /* 3. parameter mean over workers */
    for (int64_t j = 0; j < N; ++j) {
        double s = 0.0;
        for (int i = 0; i < W; ++i) s += theta[(int64_t)i * N + j];
        theta_avg[j] = s / (double)W;
    }

    /* 4. SlowMo outer momentum against the reference model */
    for (int64_t j = 0; j < N; ++j) {
        double delta = theta_avg[j] - theta_ref[j];
        v[j] = beta * v[j] + delta;
        theta_new[j] = theta_ref[j] + alpha * v[j];
    }

    /* 5. write the reconciled model back to every replica and the reference */
    for (int i = 0; i < W; ++i) {
        for (int64_t j = 0; j < N; ++j) theta[(int64_t)i * N + j] = theta_new[j];
    }
    for (int64_t j = 0; j < N; ++j) theta_ref[j] = theta_new[j];

    free(gbar);
    free(theta_avg);
    free(theta_new);
    return 0;
}

/* Synchronization indicator (eq. 4) with the epoch-end rule of Sec. 3.1:
 * step t (1-based within an epoch of T mini-batches) synchronizes iff
 * t mod K = 0, or t is the last mini-batch of the epoch. */
int oracle_is_sync_step(int64_t t, int64_t K, int64_t T)
{
    if (t % K == 0) return 1;
    if (t == T) return 1;
    return 0;
}

/* Learning rate of the training protocol at 0-based global step s (Sec. 4.3:
 * cosine annealing with linear warmup; the paper gives no formula). Reading:
 * during the first warmup_steps steps the rate rises linearly and reaches
 * base_lr on the last warmup step, lr = base_lr * (s + 1) / warmup_steps;
 * afterwards it follows one half cosine period from base_lr down towards
 * min_lr over the remaining total_steps - warmup_steps steps,
 * lr = min_lr + (base_lr - min_lr) * (1 + cos(pi * p)) / 2 with
 * p = (s - warmup_steps) / (total_steps - warmup_steps). */
double oracle_scheduled_lr(double base_lr, double min_lr, int64_t warmup_steps,
                           int64_t total_steps, int64_t s)
{
    if (s < warmup_steps) return base_lr * (double)(s + 1) / (double)warmup_steps;
    double p = (double)(s - warmup_steps) / (double)(total_steps - warmup_steps);
    return min_lr + (base_lr - min_lr) * 0.5 * (1.0 + cos(3.14159265358979323846 * p));
}

/* Synchronization indicator with the warmup rule: during the warmup epochs
 * the method runs with K = 1, i.e. every step synchronizes (Sec. 4.3, Sec. 5.4);
 * afterwards eq. 4 with the epoch-end rule. epoch is 0-based, t is 1-based. */
int oracle_is_sync_step_at(int64_t epoch, int64_t t, int64_t K, int64_t T,
                           int64_t warmup_epochs)
{
    if (epoch < warmup_epochs) return 1;
    return oracle_is_sync_step(t, K, T);
}

/* The paper's LocalSGD baseline at a synchronization step (Sec. 5.4): every
 * worker takes its own optimizer step with its own gradient, then the
 * replicas are averaged and the average written back to every worker; there
 * is no gradient averaging and no SlowMo correction, and theta_ref and v are
 * not used. Local steps between synchronizations are oracle_local_step.
 * Returns 0, or -1 if the temporary could not be allocated. */
int oracle_localsgd_sync(int W, int64_t N, double lr, double mu, double wd,
                         const double *g, double *theta, double *buf)
{
    double *theta_avg = (double *)malloc((size_t)N * sizeof(double));
    if (theta_avg == NULL) return -1;
    /* each worker's local update with its own gradient */
    for (int i = 0; i < W; ++i) {
        sgd_momentum_update(N, lr, mu, wd, g + (int64_t)i * N,
                            theta + (int64_t)i * N, buf + (int64_t)i * N);
    }
    /* parameter mean over workers, written back to every replica */
    for (int64_t j = 0; j < N; ++j) {
        double s = 0.0;
        for (int i = 0; i < W; ++i) s += theta[(int64_t)i * N + j];
        theta_avg[j] = s / (double)W;
    }
    for (int i = 0; i < W; ++i) {
        for (int64_t j = 0; j < N; ++j) theta[(int64_t)i * N + j] = theta_avg[j];
    }
    free(theta_avg);
    return 0;
}

/* The paper's DDP baseline (K = 1; Sec. 5.4, eqs. 2-3 with the optimizer of
 * Sec. 4.2): every step averages the gradients over workers and each worker
 * applies the average through its own optimizer; parameters are never
 * averaged. Returns 0, or -1 if the temporary could not be allocated. */
int oracle_ddp_step(int W, int64_t N, double lr, double mu, double wd,
                    const double *g, double *theta, double *buf)
{
    double *gbar = (double *)malloc((size_t)N * sizeof(double));
    if (gbar == NULL) return -1;
    for (int64_t j = 0; j < N; ++j) {
        double s = 0.0;
        for (int i = 0; i < W; ++i) s += g[(int64_t)i * N + j];
        gbar[j] = s / (double)W;
    }
    for (int i = 0; i < W; ++i) {
        sgd_momentum_update(N, lr, mu, wd, gbar,
                            theta + (int64_t)i * N, buf + (int64_t)i * N);
    }
    free(gbar);
    return 0;
}

/* One AdamW step of one worker (the optimizer of the paper's ViT-S runs,
 * Sec. 5.2 and Table 3: AdamW with decoupled weight decay; moments stay per
 * worker, Sec. 4.2). Written from the algorithm's definition (decoupled weight
 * decay, first and second moment estimates with bias correction), with
 * step = the 1-based number of optimizer steps taken so far:
 *   theta = theta - lr * wd * theta
 *   m = beta1 * m + (1 - beta1) * g;   s = beta2 * s + (1 - beta2) * g * g
 *   m_hat = m / (1 - beta1^step);       s_hat = s / (1 - beta2^step)
 *   theta = theta - lr * m_hat / (sqrt(s_hat) + eps)                          */
static void adamw_update(int64_t N, double lr, double beta1, double beta2, double eps,
                         double wd, int64_t step, const double *grad, double *theta,
                         double *m, double *s)
{
    double bc1 = 1.0 - pow(beta1, (double)step);
    double bc2 = 1.0 - pow(beta2, (double)step);
    for (int64_t j = 0; j < N; ++j) {
        theta[j] = theta[j] - lr * wd * theta[j];
        m[j] = beta1 * m[j] + (1.0 - beta1) * grad[j];
        s[j] = beta2 * s[j] + (1.0 - beta2) * grad[j] * grad[j];
        double m_hat = m[j] / bc1;
        double s_hat = s[j] / bc2;
        theta[j] = theta[j] - lr * m_hat / (sqrt(s_hat) + eps);
    }
}

/* Local update phase with AdamW: every worker steps with its own gradient. */
void oracle_adamw_local_step(int W, int64_t N, double lr, double beta1, double beta2,
                             double eps, double wd, int64_t step, const double *g,
                             double *theta, double *m, double *s)
{
    for (int i = 0; i < W; ++i) {
        adamw_update(N, lr, beta1, beta2, eps, wd, step, g + (int64_t)i * N,
                     theta + (int64_t)i * N, m + (int64_t)i * N, s + (int64_t)i * N);
    }
}

/* Synchronization phase with AdamW as the optimizer: the same five stages as
 * oracle_reconcile (gradient mean, every worker's own AdamW step with it,
 * parameter mean, SlowMo, write-back); both moment buffers stay per worker.
 * Returns 0, or -1 if the temporaries could not be allocated. */
int oracle_adamw_reconcile(int W, int64_t N, double lr, double beta1, double beta2,
                           double eps, double wd, int64_t step, double beta, double alpha,
                           const double *g, double *theta, double *m, double *s,
                           double *theta_ref, double *v)
{
    double *gbar = (double *)malloc((size_t)N * sizeof(double));
    double *theta_avg = (double *)malloc((size_t)N * sizeof(double));
    double *theta_new = (double *)malloc((size_t)N * sizeof(double));
    if (gbar == NULL || theta_avg == NULL || theta_new == NULL) {
        free(gbar);
        free(theta_avg);
        free(theta_new);
        return -1;
    }
    for (int64_t j = 0; j < N; ++j) {
        double acc = 0.0;
        for (int i = 0; i < W; ++i) acc += g[(int64_t)i * N + j];
        gbar[j] = acc / (double)W;
    }
    for (int i = 0; i < W; ++i) {
        adamw_update(N, lr, beta1, beta2, eps, wd, step, gbar, theta + (int64_t)i * N,
                     m + (int64_t)i * N, s + (int64_t)i * N);
    }
    for (int64_t j = 0; j < N; ++j) {
        double acc = 0.0;
        for (int i = 0; i < W; ++i) acc += theta[(int64_t)i * N + j];
        theta_avg[j] = acc / (double)W;
    }
    for (int64_t j = 0; j < N; ++j) {
        double delta = theta_avg[j] - theta_ref[j];
        v[j] = beta * v[j] + delta;
        theta_new[j] = theta_ref[j] + alpha * v[j];
    }
    for (int i = 0; i < W; ++i) {
        for (int64_t j = 0; j < N; ++j) theta[(int64_t)i * N + j] = theta_new[j];
    }
    for (int64_t j = 0; j < N; ++j) theta_ref[j] = theta_new[j];
    free(gbar);
    free(theta_avg);
    free(theta_new);
    return 0;
}

/* The LocalSGD baseline's synchronization step (Sec. 5.4) with AdamW as the
 * workers' optimizer: every worker's own AdamW step with its own gradient,
 * then the parameter mean written back to every replica. */
int oracle_adamw_localsgd_sync(int W, int64_t N, double lr, double beta1, double beta2,
                               double eps, double wd, int64_t step, const double *g,
                               double *theta, double *m, double *s)
{
    double *theta_avg = (double *)malloc((size_t)N * sizeof(double));
    if (theta_avg == NULL) return -1;
    for (int i = 0; i < W; ++i) {
        adamw_update(N, lr, beta1, beta2, eps, wd, step, g + (int64_t)i * N,
                     theta + (int64_t)i * N, m + (int64_t)i * N, s + (int64_t)i * N);
    }
    for (int64_t j = 0; j < N; ++j) {
        double acc = 0.0;
        for (int i = 0; i < W; ++i) acc += theta[(int64_t)i * N + j];
        theta_avg[j] = acc / (double)W;
    }
    for (int i = 0; i < W; ++i) {
        for (int64_t j = 0; j < N; ++j) theta[(int64_t)i * N + j] = theta_avg[j];
    }
    free(theta_avg);
    return 0;
}

/* The DDP baseline's step (Sec. 5.4, eqs. 2-3) with AdamW: the gradient mean,
 * then every worker's own AdamW step with it; no parameter mean. */
int oracle_adamw_ddp_step(int W, int64_t N, double lr, double beta1, double beta2,
                          double eps, double wd, int64_t step, const double *g,
                          double *theta, double *m, double *s)
{
    double *gbar = (double *)malloc((size_t)N * sizeof(double));
    if (gbar == NULL) return -1;
    for (int64_t j = 0; j < N; ++j) {
        double acc = 0.0;
        for (int i = 0; i < W; ++i) acc += g[(int64_t)i * N + j];
        gbar[j] = acc / (double)W;
    }
    for (int i = 0; i < W; ++i) {
        adamw_update(N, lr, beta1, beta2, eps, wd, step, gbar, theta + (int64_t)i * N,
                     m + (int64_t)i * N, s + (int64_t)i * N);
    }
    free(gbar);
    return 0;
}

/* Optimizer-state reconciliation, the variant the paper names but does not
 * use (Sec. 4.2, on optimizer state; Sec. 6, future work).
 * Reading: after a synchronization step's optimizer updates, one per-worker
 * state array (the momentum buffers, or each AdamW moment) is replaced on
 * every worker by its mean over the workers. */
int oracle_average_state(int W, int64_t N, double *state)
{
    double *mean = (double *)malloc((size_t)N * sizeof(double));
    if (mean == NULL) return -1;
    for (int64_t j = 0; j < N; ++j) {
        double acc = 0.0;
        for (int i = 0; i < W; ++i) acc += state[(int64_t)i * N + j];
        mean[j] = acc / (double)W;
    }
    for (int i = 0; i < W; ++i) {
        for (int64_t j = 0; j < N; ++j) state[(int64_t)i * N + j] = mean[j];
    }
    free(mean);
    return 0;
}
