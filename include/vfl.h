/*
 * vfl.h -- C ABI of the GB300 split-VFL training step (PubSub-VFL, arxiv 2510.12494).
 *
 * The library runs the two-party split-learning training step of the paper on
 * one GPU: the passive party's bottom MLP forward publishes its embedding into a
 * device-side channel, the active party runs its bottom MLP, the top MLP on
 * [z^a | z^p], the loss and the backward pass, publishes the embedding gradient
 * back, and both parties apply SGD (paper Sec. 3, Eq. 1-2; Algorithm 1).  The
 * weight versions each step consumes come from a staleness schedule (the
 * delayed update of App. D, Assumption 4).
 *
 * Conventions shared by every entry point:
 *  - Every function returns a vfl_status and never throws.  On failure the
 *    context keeps a message readable through vfl_last_error().
 *  - Matrices are row-major.  A Linear layer with `in` inputs and `out`
 *    outputs has W [out, in] and b [out], and computes Y = X W^T + b.
 *  - Party ids: 0 = passive bottom f_p (theta_2), 1 = active bottom f_a,
 *    2 = top model g (1 and 2 together are theta_1).
 *  - "Host pointer" arguments are read or written before the call returns
 *    (except vfl_fetch_loss and the arrays bound by vfl_bind_host_data, which
 *    are used asynchronously); the caller keeps ownership.
 *  - Device memory comes from the caller: vfl_workspace_bytes() says how much,
 *    vfl_create() carves every device buffer out of that one allocation.
 *  - Work is enqueued on caller-provided CUDA streams (vfl_set_streams);
 *    without them the library uses the legacy default stream for every worker.
 *  - After VFL_E_CUDA the context is unusable except for vfl_destroy().
 */
#ifndef VFL_H
#define VFL_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int32_t vfl_status;

#define VFL_OK 0
#define VFL_E_INVAL 1     /* bad argument (shape, range, null pointer)                  */
#define VFL_E_OOM 2       /* workspace smaller than vfl_workspace_bytes()               */
#define VFL_E_CUDA 3      /* a CUDA call failed; the context is now unusable            */
#define VFL_E_STATE 4     /* call out of order (step ordering / staleness contract)    */
#define VFL_E_VERSION 5   /* a subscriber found a channel header for another step      */
#define VFL_E_TIMEOUT 6   /* a bounded device-side wait gave up                         */

#define VFL_MAX_LAYERS 8

#define VFL_LOSS_BCE 0    /* binary cross-entropy on one logit (Eq. 1)                  */
#define VFL_LOSS_CE 1     /* softmax cross-entropy on n_out >= 2 logits                */

#define VFL_FP32 0        /* fp32 storage and arithmetic                               */
#define VFL_BF16 1        /* bf16 weights copies / activations, fp32 accumulate+master */

#define VFL_DP_GRAD 0     /* DP on the published embedding gradient dLoss/dz^p          */
#define VFL_DP_EMB 1      /* DP on the published embedding z^p (App. C)                 */

#define VFL_SCHED_SYNC 0  /* tau = 0                                                    */
#define VFL_SCHED_MAX 1   /* tau(k) = min(k, S)                                         */
#define VFL_SCHED_SEEDED 2

/* what vfl_tap() reads */
#define VFL_TAP_EMB 0     /* published embedding z^p of step k, [B_k, e_p]              */
#define VFL_TAP_GRAD 1    /* published gradient dLoss/dz^p of step k, [B_k, e_p]        */
#define VFL_TAP_LOGITS 2  /* logits of the last active step run on k's worker, [B_k, n_out] */
#define VFL_TAP_ZA 3      /* active embedding z^a of that step, [B_k, e_a]              */
#define VFL_TAP_DZA 4     /* dLoss/dz^a of that step, [B_k, e_a]                        */
/* the output of Linear+ReLU layer `layer` of `party` for step k, [B_k, width] (per-layer kernels only:
 * VFL_E_STATE on a context that runs the fused fp32 kernels): party 0 = f_p (its last layer is z^p before
 * any DP), 1 = f_a, 2 = the hidden layers of g */
#define VFL_TAP_ACT(party, layer) (16 + 16 * (party) + (layer))

typedef struct vfl_config {
    int32_t d_passive;                      /* passive feature count d_p                 */
    int32_t d_active;                       /* active feature count d_a                  */
    int32_t n_passive, n_active, n_top;     /* Linear layers in f_p, f_a, g (1..8)       */
    int32_t passive_out[VFL_MAX_LAYERS];    /* output width of each f_p layer            */
    int32_t active_out[VFL_MAX_LAYERS];     /* output width of each f_a layer            */
    int32_t top_out[VFL_MAX_LAYERS];        /* output width of each g layer; last = n_out */
    int32_t loss;                           /* VFL_LOSS_BCE (n_out == 1) | VFL_LOSS_CE   */
    int32_t dtype;                          /* VFL_FP32 | VFL_BF16                       */
    int32_t batch;                          /* rows per step B (the last batch may be shorter) */
    float lr;                               /* SGD step size eta (Eq. 2)                 */
    int32_t staleness;                      /* bound S on tau; channels hold S+1 slots   */
    int32_t workers;                        /* worker streams per party (1..16)          */
    float dp_clip;                          /* > 0 enables DP on the tensor dp_target names */
    float dp_sigma;                         /* noise multiplier; noise std = sigma * clip */
    uint64_t dp_seed;                       /* Philox key of the DP noise                */
    int32_t dp_target;                      /* VFL_DP_GRAD | VFL_DP_EMB (see below)       */
    int32_t ps_dt0;                         /* > 0: intra-party parameter server, Delta T_0 (see below) */
} vfl_config;

/*
 * DP mechanisms (App. C), both per row of the batch, with N(0,1) draws from
 * Philox4x32-10 keyed by dp_seed (counter (col / 4, row, k, tag), Box-Muller):
 *  - VFL_DP_GRAD: the published gradient, g_i = B_k dz_i clipped to L2 norm C,
 *    plus sigma C xi_i, divided by B_k (tag 0x4450);
 *  - VFL_DP_EMB: the published embedding, c_i = min(1, C / ||z_i||) (1 for a
 *    zero row), published c_i z_i + sigma C xi_i (tag 0x4445); the passive
 *    backward scales the gradient it receives by c_i before its ReLU mask on
 *    the clean z (straight-through: the Jacobians of c_i and the noise are
 *    ignored).
 * Either sends the model through the per-layer kernels.
 */

/*
 * Intra-party semi-asynchronous parameter server (Sec. 4.1, Eq. 5), enabled by
 * ps_dt0 > 0 (requires staleness == 0).  Each party keeps one replica of its
 * parameters (fp32 master and compute copy) per worker; step k runs on worker
 * w = k mod workers, reads replica w as it stands and applies its SGD update to
 * replica w only, so the workers' chains run concurrently on their own stream
 * pairs.  After the last step of epoch t (t = 1, 2, ...; an epoch is
 * ceil(n_rows / batch) steps) every party's replicas are replaced by their mean
 * (fp32 sum over the workers in order 0..W-1, then divided by W) when
 * t mod Delta T_t == 0, Delta T_t = ceil(Delta T_0 / 2 tanh(2 t / Delta T_0 - 2)
 * + Delta T_0 / 2).  vfl_get_params reads replica 0; vfl_get_replica /
 * vfl_set_replica read and write any replica (they replace the version API,
 * which answers VFL_E_STATE in this mode).
 */

/* Delta T_t of Eq. 5 for epoch t >= 1 and Delta T_0 = dt0 >= 1 (host only, pure): the
 * parameter-server mode averages the replicas after epoch t when t mod Delta T_t == 0.
 * VFL_E_INVAL for t < 1, dt0 < 1 or a null output. */
vfl_status vfl_ps_interval(int64_t t, int32_t dt0, int64_t* interval);

/* Noise multiplier for mu-GDP on the published embedding, Eq. 25 with the O(.)
 * constant taken as 1: sigma = batch sqrt(queries) / (mu n_rows), queries = the
 * batches the worker processes.  VFL_E_INVAL unless mu > 0, batch >= 1,
 * n_rows >= 1 and queries >= 1. */
vfl_status vfl_gdp_sigma(double mu, int64_t batch, int64_t n_rows, int64_t queries, double* sigma);

/*
 * System planning (Sec. 4.2-4.3, Eq. 7-17, Algorithm 2).  Host only, pure.
 * Delay model of one iteration, each term coef * B^exp * w / C (Eq. 7-9):
 *   T_A = (lambda_a B^gamma_a + phi_a B^beta_a + lambda_top B^gamma_top + phi_top B^beta_top) w_a / C_a
 *   T_P = (lambda_p B^gamma_p + phi_p B^beta_p) w_p / C_p
 *   O(w_a, w_p, B) = max(T_A, T_P) + (E + G) / B_b,  E = G = B * bytes_per_row   (Eq. 10, 17)
 * Memory per worker M(B) = M0 + rho B^chi, so B <= B_max = min over the two parties of
 * ((M_max - M0) / rho)^(1/chi) (Eq. 14-15; a party with rho <= 0 sets no bound).
 */
typedef struct vfl_plan_model {
    double lambda_a, gamma_a, phi_a, beta_a;          /* active bottom forward / backward        */
    double lambda_top, gamma_top, phi_top, beta_top;  /* top model forward / backward (Eq. 9)    */
    double lambda_p, gamma_p, phi_p, beta_p;          /* passive bottom forward / backward       */
    double C_a, C_p;                                  /* compute units of each party (> 0)       */
    double bytes_per_row;                             /* cut-layer payload per row, each direction */
    double bandwidth;                                 /* B_b (> 0), bytes per time unit          */
    double M_A0, rho_A, M_A_max;                      /* active memory model per worker          */
    double M_P0, rho_P, M_P_max;                      /* passive memory model per worker         */
    double chi;                                       /* memory exponent (> 0)                   */
} vfl_plan_model;

/* B_max of Eq. 15 (+inf when neither party bounds it; VFL_E_INVAL when a bound is negative). */
vfl_status vfl_plan_bmax(const vfl_plan_model* m, double* bmax);

/* O(w_a, w_p, B) of Eq. 17 for one configuration. */
vfl_status vfl_plan_delay(const vfl_plan_model* m, int32_t w_a, int32_t w_p, double batch, double* delay);

/*
 * Algorithm 2: the (w_a, w_p, B) minimising O over w_a in [wa_lo, wa_hi], w_p in
 * [wp_lo, wp_hi] and the candidate batches (n_batches of them) with B <= B_max.
 * Scan order: batches as given, then w_a, then w_p ascending; the first strict
 * minimum wins.  VFL_E_INVAL when no candidate is feasible or a range is empty.
 */
vfl_status vfl_plan(const vfl_plan_model* m, int32_t wa_lo, int32_t wa_hi, int32_t wp_lo, int32_t wp_hi,
                    const int32_t* batches, int32_t n_batches, int32_t* w_a, int32_t* w_p, int32_t* batch,
                    double* delay);

/* Least-squares fit of t = coef * x^expo in log space over n >= 2 points (x, t > 0, not all x equal):
 * the profiling step that turns measured delays into the constants of Eq. 7-9. */
vfl_status vfl_fit_power(const double* x, const double* t, int32_t n, double* coef, double* expo);

typedef struct vfl_ctx vfl_ctx;

/* Bytes of device workspace vfl_create() needs for `cfg` and a dataset of n_rows rows: both parties'
 * feature partitions and the labels (Sec. 3), the S+1 weight versions each party keeps (App. D,
 * Assumption 4), the embedding and gradient channel buffers (Sec. 4.1) and the per-worker scratch. */
vfl_status vfl_workspace_bytes(const vfl_config* cfg, int64_t n_rows, uint64_t* bytes);

/*
 * Create a context on the current CUDA device for the problem of Sec. 3: the passive party's d_p
 * features and bottom model f_p, the active party's d_a features, labels, bottom model f_a and top
 * model g, the loss (Eq. 1 for BCE), the step size of Eq. 2, the staleness bound of App. D
 * (Assumption 4), the channels of Sec. 4.1 (S+1 slots each) and the workers per party (Fig. 2).
 * VFL_E_INVAL for a configuration outside the limits above, VFL_E_OOM for a short workspace.  `workspace` is a device pointer
 * (256-byte aligned) of at least vfl_workspace_bytes() bytes; it stays owned by
 * the caller and must outlive the context.  Parameters start at zero: set them
 * with vfl_set_params() before training.
 */
vfl_status vfl_create(const vfl_config* cfg, int64_t n_rows, void* workspace, uint64_t workspace_bytes,
                      vfl_ctx** out);
/* Release the context (the paper has no counterpart).  Waits for its work; the workspace and the
 * borrowed streams stay the caller's.  Valid in every state, including after VFL_E_CUDA. */
vfl_status vfl_destroy(vfl_ctx* ctx);

/*
 * The workers of each party (Sec. 4.1, Fig. 2: each party runs several workers that publish and
 * subscribe concurrently) are CUDA streams here.
 * Borrow 2*workers CUDA streams (cudaStream_t passed as void*): entries
 * [0, workers) run the passive party's work, [workers, 2*workers) the active
 * party's.  Steps go to worker k mod workers.  The streams must outlive the context.
 */
vfl_status vfl_set_streams(vfl_ctx* ctx, int32_t n, void* const* streams);

/*
 * The vertically partitioned dataset of Sec. 3: the passive party holds x^p, the active party x^a
 * and the labels y, row i of each belonging to the same sample (rows aligned by construction).
 * Copy the whole dataset from host memory: x_passive [n_rows, d_p] and
 * x_active [n_rows, d_a] fp32, y [n_rows] int32 (BCE: 0/1, CE: class id in
 * [0, n_out)).  Synchronous.  bf16 contexts round the features to bf16 here.
 */
vfl_status vfl_load_data(vfl_ctx* ctx, const float* x_passive, const float* x_active, const int32_t* y);

/*
 * Host-resident data (the same partitioned dataset of Sec. 3, left in host memory; the paper has no
 * counterpart for the staging).  After this call every step k reads its own rows
 * [r0, r1) of x_passive [n_rows, d_p] fp32, x_active [n_rows, d_a] fp32 and
 * y [n_rows] int32 straight from host memory into a device staging ring of
 * S + workers + 2 slots (part of the workspace), with one kernel on io_stream
 * (or, when the arrays are page-locked and already in the slots' layout -- the
 * context's dtype, d_p and d_a multiples of 8 -- with three copies by the copy
 * engines, which leave the SMs to the steps' kernels), and its phases read the
 * rows there; the kernel that computes the step's mean
 * loss also writes it to loss_out[k mod loss_cap] (skipped when loss_out is
 * null).  A step's rows are read once the step that last used its slot has
 * finished both updates.  The arrays must be page-locked (cudaHostAlloc,
 * cudaHostRegister; VFL_E_INVAL otherwise) unless the device accesses pageable
 * memory through the host's page tables, and must stay valid while steps that
 * use them are in flight or a graph captured under the binding can still be
 * launched: graphs captured under it contain the staging, and launch only
 * while it holds.  io_stream is a caller stream (not a worker stream) that must
 * outlive the binding.  The labels are checked here as vfl_load_data checks
 * them; bf16 contexts round the staged rows to bf16.  Pass x_passive = null to
 * unbind (the device-resident dataset is used again).  Valid only while no step
 * is in flight; synchronizes the context.
 */
vfl_status vfl_bind_host_data(vfl_ctx* ctx, const float* x_passive, const float* x_active, const int32_t* y,
                              float* loss_out, int64_t loss_cap, void* io_stream);

/*
 * The same binding for a bf16 context whose host dataset is already in its compute dtype (the same
 * partitioned dataset of Sec. 3; no counterpart in the paper): x_passive [n_rows, d_p] and
 * x_active [n_rows, d_a] hold bf16 bit patterns (round-to-nearest-even of the fp32 features gives the
 * rows vfl_load_data would store), y [n_rows] int32; VFL_E_INVAL for an fp32 context.  Each step's
 * staging kernel then copies its rows without rounding: half the bytes over the host link of the fp32
 * binding.  Everything else is as for vfl_bind_host_data; x_passive = null unbinds.
 */
vfl_status vfl_bind_host_data_bf16(vfl_ctx* ctx, const uint16_t* x_passive, const uint16_t* x_active,
                                   const int32_t* y, float* loss_out, int64_t loss_cap, void* io_stream);

/*
 * The same binding for binary features (every feature 0 or 1, as in a party's indicator columns of the
 * partitioned dataset of Sec. 3; no counterpart in the paper), held bit-packed on the host:
 * x_passive [n_rows, ceil(d_p / 32)] and x_active [n_rows, ceil(d_a / 32)] uint32 words, feature c of a
 * row in bit (c mod 32) of the row's word c / 32 (bits past d in a row's last word are ignored);
 * y [n_rows] int32.  Each step's staging kernel reads its rows' words and writes the values 1 / 0 into
 * the staging slot in the context's dtype (bf16 or fp32): 1/16 of the host-link bytes of bf16 rows, and
 * exact, so the steps are bit-identical to a binding of the same features as fp32 or bf16 rows.
 * Everything else (page-locked arrays, io_stream, labels, loss_out, graphs) is as for
 * vfl_bind_host_data; x_passive = null unbinds.
 */
vfl_status vfl_bind_host_data_bits(vfl_ctx* ctx, const uint32_t* x_passive, const uint32_t* x_active,
                                   const int32_t* y, float* loss_out, int64_t loss_cap, void* io_stream);

/*
 * The parameters theta_2 (f_p) and theta_1 (f_a and g) of Sec. 3 that Eq. 2 updates.
 * Set / read the fp32 master parameters of one layer: W [out, in], b [out]
 * (host pointers).  vfl_set_params resets every stored weight version of the
 * layer to the new values and is only valid before the first step.
 * vfl_get_params synchronizes the context first.
 */
vfl_status vfl_set_params(vfl_ctx* ctx, int32_t party, int32_t layer, const float* W, const float* b);
vfl_status vfl_get_params(vfl_ctx* ctx, int32_t party, int32_t layer, float* W, float* b);

/*
 * Algorithm 1 starts from random weights theta_1, theta_2 without naming a distribution; this
 * library's reading is a uniform fan-in draw.
 * Seeded initial parameters for every layer, as vfl_set_params would take them: each entry of
 * layer l of party q (W row-major, then b) is (2u - 1) / sqrt(fan_in) in double, rounded to fp32,
 * u = word i * 2^-32 of the stream Philox4x32-10(key = (seed lo, seed hi), counter = (i / 4 lo,
 * i / 4 hi, (q << 8) | l, 0x49)) word i mod 4 -- U(-1/sqrt(fan_in), 1/sqrt(fan_in)).  Only valid
 * before the first step.
 */
vfl_status vfl_init_params(vfl_ctx* ctx, uint64_t seed);

/*
 * The gradients grad_theta_1 L and grad_theta_2 L of Sec. 3's backward pass (Eq. 2 applies them).
 * Gradient dLoss/dW [out, in] and dLoss/db [out] of one layer from the most
 * recent step of that party on worker `worker` (before the SGD update used
 * it).  Synchronizes the context.
 */
vfl_status vfl_get_grads(vfl_ctx* ctx, int32_t party, int32_t layer, int32_t worker, float* dW, float* db);

/*
 * Checkpoint / restore of the state the delayed update of App. D reads: the step counter and the
 * stored weight versions theta^(k - tau), tau <= S (the paper has no checkpoint format).
 * Valid only while no step is in flight (every enqueued
 * step has run all three phases).
 *  - vfl_step_cursor: number of finished steps k = the current weight version.
 *  - vfl_get_version: the stored compute copy of weight version v
 *    (max(0, k-S) <= v <= k) as fp32 (exact: bf16 copies widen losslessly).
 *  - vfl_set_cursor: make k the next step (for resuming a checkpoint); the
 *    caller then stores versions max(0, k-S) .. k with vfl_set_version.
 *  - vfl_set_version: store version v of one layer (rounded to the compute
 *    dtype); for v == k it also sets the fp32 master that SGD updates.
 * The fp32 master of version k is read with vfl_get_params.  A context
 * restored this way continues bit-identically to the one checkpointed.
 */
vfl_status vfl_step_cursor(vfl_ctx* ctx, int64_t* k);
vfl_status vfl_get_version(vfl_ctx* ctx, int32_t party, int32_t layer, int64_t v, float* W, float* b);
vfl_status vfl_set_cursor(vfl_ctx* ctx, int64_t k);
vfl_status vfl_set_version(vfl_ctx* ctx, int32_t party, int32_t layer, int64_t v, const float* W, const float* b);

/*
 * The per-worker replicas of the intra-party parameter server (Sec. 4.1, Eq. 5).
 * Parameter-server mode only (VFL_E_STATE otherwise): the fp32 master of one
 * layer of replica `worker` (0 <= worker < workers), host pointers W [out, in]
 * and b [out].  Both synchronize the context and need no step in flight;
 * vfl_set_replica also rewrites the replica's compute copy (rounded to the
 * compute dtype).  A checkpoint in this mode is the cursor plus every replica.
 */
vfl_status vfl_get_replica(vfl_ctx* ctx, int32_t worker, int32_t party, int32_t layer, float* W, float* b);
vfl_status vfl_set_replica(vfl_ctx* ctx, int32_t worker, int32_t party, int32_t layer, const float* W, const float* b);

/*
 * Staleness schedule (host only, pure).  tau_p[k], tau_a[k] for k < n_steps:
 * SYNC 0; MAX min(k, S); SEEDED tau(0) = 0, tau(k) = min(k, S, tau(k-1)+1,
 * u_k mod (S+1)) with u_k word 0 of Philox4x32-10(key = (seed lo, seed hi),
 * counter = (k lo, k hi, party, 0x5343)).  Paper: App. D Assumption 4 bounds the
 * delay; the seeded draw is this library's schedule.
 */
vfl_status vfl_make_schedule(uint64_t seed, int32_t S, int32_t kind, int64_t n_steps, int32_t* tau_p,
                             int32_t* tau_a);

/*
 * Publisher phase of step k (Algorithm 1, passive): z^p = f_p(x^p) with the
 * passive weights of version k - tau_p, then publish z^p to the embedding
 * channel slot k mod (S+1) with header {k, batch, version}.  Steps must be
 * published in order (k = number of earlier calls); the version must still be
 * stored: 0 <= tau_p <= min(k, S) and k - tau_p >= (passive updates so far) - S.
 */
vfl_status vfl_passive_forward(vfl_ctx* ctx, int64_t k, int32_t tau_p);

/*
 * Subscriber phase of step k (Algorithm 1, active): fetch z^p (header check,
 * VFL_E_VERSION on mismatch), z^a = f_a(x^a) and y_hat = g(z^a, z^p) with the
 * active+top weights of version k - tau_a, loss, backward, optional DP on the
 * gradient, publish dLoss/dz^p to the gradient channel, then the SGD update of
 * f_a and g (Eq. 2, applied in step order).  Requires the embedding of step k
 * to have been enqueued.
 */
vfl_status vfl_active_step(vfl_ctx* ctx, int64_t k, int32_t tau_a);

/*
 * Backward phase of step k (Algorithm 1, passive): fetch dLoss/dz^p (header
 * check), backward through the passive version used by the forward of step k
 * with its saved activations, SGD update of f_p in step order.
 */
vfl_status vfl_passive_backward(vfl_ctx* ctx, int64_t k);

/*
 * Waiting deadline / buffer overflow (Sec. 4.1; Algorithm 1's subscriber branch):
 * the subscriber of step k gives up on its embedding (it did not arrive within
 * the deadline, or a full buffer discarded it oldest-first).  Called instead of
 * vfl_active_step(k): step k trains nothing, records a NaN loss, and both
 * parties' version k+1 equals version k; vfl_passive_backward(k) is still called
 * (the passive party is notified: it skips its backward and carries its version
 * forward).  The batch of step k is reassigned to step k+1: step k trains batch
 * (k - D) mod nb, D the drops before k.  Valid when step k is the next active
 * step and no later step has been published (its batch would change); if step
 * k was never published, its publish is skipped.
 * vfl_get_drops / vfl_set_drops read and (with no step in flight, for restoring
 * a checkpoint after vfl_set_cursor) set D for the next step.
 */
vfl_status vfl_drop_step(vfl_ctx* ctx, int64_t k);
vfl_status vfl_get_drops(vfl_ctx* ctx, int64_t* n_drops);
vfl_status vfl_set_drops(vfl_ctx* ctx, int64_t n_drops);

/*
 * Seeded drop draws for the waiting-deadline / buffer-overflow drops of Sec. 4.1
 * (host only, pure): drop[k] = 1 when word 0 of
 * Philox4x32-10(key = (seed lo, seed hi), counter = (k lo, k hi, 2, 0x4452)) is
 * below floor(rate * 2^32) (every step when rate == 1).  VFL_E_INVAL unless
 * 0 <= rate <= 1.
 */
vfl_status vfl_make_drops(uint64_t seed, double rate, int64_t n_steps, uint8_t* drop);

/*
 * Algorithm 1's three phases (publisher, subscriber, backward) for a window of steps, each step's
 * versions fixed by the staleness schedule (App. D).
 * Enqueue steps [k0, k0 + n_steps) as one dependency graph across the worker
 * streams: each publisher phase runs as soon as its weight version exists, so
 * the parties overlap as far as tau allows.  tau_p / tau_a are host arrays
 * indexed by absolute step (length >= k0 + n_steps).  `drop` (NULL: none) marks
 * the steps whose subscriber gives up (see vfl_drop_step), indexed the same way.
 * Same contract as the per-phase calls.
 */
vfl_status vfl_train_steps(vfl_ctx* ctx, int64_t k0, int64_t n_steps, const int32_t* tau_p,
                           const int32_t* tau_a, const uint8_t* drop);

/*
 * CUDA-graph replay of a window of steps (the paper has no counterpart: the same phases of
 * Algorithm 1 as vfl_train_steps, recorded once and replayed).  vfl_graph_capture records steps
 * [k0, k0 + n_steps) -- the same kernels and cross-stream events
 * vfl_train_steps would enqueue -- into an executable graph without running
 * them; every step before k0 must be enqueued (it may still be running, e.g. a
 * replayed graph: the host can capture the next window meanwhile) and the
 * cursor stays at k0.
 * vfl_graph_launch replays it once (the context must be at cursor k0), ordered
 * after all work already on the context's streams, and advances the cursor to
 * k0 + n_steps.  Capture needs caller streams (vfl_set_streams) and per-launch
 * timing off.  A graph belongs to one context; destroy it before the context.
 * `drop` as for vfl_train_steps; the batches are baked in, so a replay also
 * needs the drop count the capture started from.
 */
typedef struct vfl_graph vfl_graph;
vfl_status vfl_graph_capture(vfl_ctx* ctx, int64_t k0, int64_t n_steps, const int32_t* tau_p,
                             const int32_t* tau_a, const uint8_t* drop, vfl_graph** out);
vfl_status vfl_graph_launch(vfl_ctx* ctx, vfl_graph* graph);

/*
 * (No counterpart in the paper; an update of a vfl_graph_capture graph.)
 * Re-record `graph` for steps [k0, k0 + n_steps) (same preconditions as vfl_graph_capture) and update
 * its executable graph in place (cudaGraphExecUpdate): far cheaper than a new capture's
 * instantiation when the new window has the same shape.  Launches already in flight keep their old
 * contents.  VFL_E_STATE when the shape differs (the graph is then unchanged and still replays its
 * old window); windows of one length have one shape in the uniform order (vfl_set_order) without
 * drops or parameter-server averaging.
 */
vfl_status vfl_graph_update(vfl_ctx* ctx, vfl_graph* graph, int64_t k0, int64_t n_steps, const int32_t* tau_p,
                            const int32_t* tau_a, const uint8_t* drop);

/*
 * Dependency order of the enqueued steps (no counterpart in the paper: both orders compute what
 * App. D's delayed update defines).  VFL_ORDER_OVERLAP (default): a step waits only for the
 * version it reads, so steps overlap as far as tau allows.  VFL_ORDER_UNIFORM: every step waits for
 * all updates before it and is published after the previous backward, as if tau were 0, while
 * still computing with versions k - tau -- the same results, less overlap, but one graph shape for
 * every window (vfl_graph_update).  Only with no step in flight.
 */
#define VFL_ORDER_OVERLAP 0
#define VFL_ORDER_UNIFORM 1
vfl_status vfl_set_order(vfl_ctx* ctx, int32_t order);
vfl_status vfl_graph_destroy(vfl_graph* graph);

/* Wait for all enqueued work (no counterpart in the paper); returns VFL_E_VERSION (a channel header
 * of Sec. 4.1 named another step) or VFL_E_TIMEOUT recorded by kernels. */
vfl_status vfl_synchronize(vfl_ctx* ctx);

/* The loss of Eq. 1 (BCE) or softmax cross-entropy, averaged over each step's rows: steps
 * [k0, k0+n) (float per step, NaN for a dropped step) into host memory; synchronizes.
 * Only the last 4096 steps are kept. */
vfl_status vfl_read_losses(vfl_ctx* ctx, int64_t k0, int64_t n, float* out);

/*
 * Algorithm 1's epoch loop (global epoch t: every batch B_j once, through the three phases).
 * One epoch: steps [epoch * nb, (epoch + 1) * nb) (nb = ceil(n_rows / batch)) through
 * vfl_train_steps (same arrays, indexed by absolute step; `drop` may be NULL) -- in the uniform order
 * (vfl_set_order) without drops, as a CUDA graph the context keeps per epoch shape and updates in
 * place for every later epoch (vfl_graph_update) -- then, when
 * mean_loss_out is not NULL, a synchronize and the epoch's mean loss per sample: each trained
 * step's mean loss weighted by its rows (dropped steps count none).  The steps before the epoch
 * must all be enqueued.
 */
vfl_status vfl_train_epoch(vfl_ctx* ctx, int64_t epoch, const int32_t* tau_p, const int32_t* tau_a,
                           const uint8_t* drop, float* mean_loss_out);

/*
 * The loss of Eq. 1 for one step, read without a synchronisation.
 * Enqueue an asynchronous copy of the mean loss of step k (already enqueued)
 * into host memory `host_out` (pinned for asynchrony) on the stream of the
 * step's active worker; valid once that stream passes this point.
 */
vfl_status vfl_fetch_loss(vfl_ctx* ctx, int64_t k, float* host_out);

/* Parity probe of Algorithm 1's exchanged tensors (z^p in C_e[B_j], grad_z^p L in C_g[B_j]) and of
 * the active party's z^a, grad_z^a L and logits (Sec. 3).
 * Copy a channel slot or a per-worker buffer of step k to host fp32 (see VFL_TAP_*): rows x cols
 * floats, rows as vfl_step_rows gives; VFL_E_INVAL when that exceeds out_elems.  Synchronizes. */
vfl_status vfl_tap(vfl_ctx* ctx, int64_t k, int32_t what, float* out, int64_t out_elems);

/* Batch B_j of step k (Algorithm 1's sampled batch; its id labels the channels, Sec. 4.1).
 * First row and row count of the batch step k trains (published steps in flight, or the next
 * step): batch (k - drops before k) mod nb. */
vfl_status vfl_step_rows(vfl_ctx* ctx, int64_t k, int64_t* r0, int32_t* rows);

/*
 * Sec. 4.1's waiting deadline T_ddl as a device-side probe.
 * Fault probe: a bounded device-side wait (at most max_iters polls) for the
 * embedding (which = 0) or gradient (which = 1) channel slot of step k to carry
 * header k.  Returns VFL_OK or VFL_E_TIMEOUT; never blocks indefinitely.
 */
vfl_status vfl_wait_channel(vfl_ctx* ctx, int32_t which, int64_t k, int64_t max_iters);

/*
 * Sec. 4.1's batch-ID labelled channels: the subscriber's check of the slot's label.
 * Non-blocking subscriber check: does the embedding (which = 0) or gradient
 * (which = 1) channel slot of step k carry the header of step k?  VFL_OK or
 * VFL_E_VERSION (the same device-side check the subscriber phases run).
 * Synchronizes the context.
 */
vfl_status vfl_check_channel(vfl_ctx* ctx, int32_t which, int64_t k);

/* Number of kernels this context has launched so far (launch accounting; no counterpart in the paper). */
int64_t vfl_kernel_launches(const vfl_ctx* ctx);

/* Communication cost (Sec. 5's metric): payload bytes published so far through the embedding and
 * gradient channels (B_k x e_p elements of the compute dtype per publish; a dropped step publishes
 * its embedding, if its publisher ran, and no gradient).  Host counters, no synchronisation. */
vfl_status vfl_exchange_bytes(const vfl_ctx* ctx, int64_t* emb, int64_t* grad);

/*
 * Per-launch timing: the measurements Sec. 4.2 (System Profiling) fits the delay model of
 * Eq. 7-9 to.  vfl_profile(ctx, 1) starts recording a CUDA event pair
 * around every kernel launch, on the launch's stream; vfl_profile(ctx, 0)
 * synchronizes and folds the records into per-class totals.  vfl_profile_get
 * then returns, for kernel class `cls` (0 .. VFL_KERNEL_CLASSES-1, named by
 * vfl_kernel_class_name), the number of launches, their summed duration in ms
 * and their summed algorithmic flops and bytes.  Launches captured into a
 * graph (vfl_graph_capture) while timing is on carry their event pairs into
 * the graph: launch it once, then call vfl_profile(ctx, 0); folding before the
 * graph has run returns VFL_E_STATE.  Such a graph should not be replayed
 * after the fold (its events go back to the context's pool).
 */
#define VFL_KERNEL_CLASSES 20
vfl_status vfl_profile(vfl_ctx* ctx, int32_t enable);
vfl_status vfl_profile_get(const vfl_ctx* ctx, int32_t cls, int64_t* launches, double* ms, double* flops,
                           double* bytes);
const char* vfl_kernel_class_name(int32_t cls);

/*
 * Weight gradient of one Linear layer without any allocation (the paper has no
 * counterpart; this is a convenience for restricted callers).
 *
 * Some callers cannot allocate device memory when they need a gradient: code
 * running inside an allocator or memory-pool callback, a host that has fixed
 * the process's device footprint in advance, or a process whose pools already
 * hold all of HBM.  This call needs no workspace: its split-K partial sums live
 * in a fixed 16 MiB array inside the library (every GPU that loads the library
 * holds it until the process exits), and it calls no cudaMalloc, cudaFree or
 * other allocating routine.
 *
 *   dpre  device [rows, out] row-major: gradient of the layer's pre-activation
 *   x     device [rows, in]  row-major: the layer's input
 *         (both float for dtype VFL_FP32, bf16 for VFL_BF16)
 *   dW    device [out, in] fp32 output: dpre^T x
 *   db    device [out] fp32 output: column sums of dpre
 *   stream  cudaStream_t to enqueue on (NULL: legacy default stream); the call
 *         returns before the work finishes.
 *
 * Limits: out*in + out <= 4,194,304 and in <= 4,194,240 (65535 blocks of 64
 * inputs); larger layers get VFL_E_INVAL with the reason in
 * vfl_last_error(NULL).  The first call on a device looks up the array's
 * device address (cudaGetSymbolAddress) and the SM count; make that first
 * call before any stream capture.  The address stays cached for the process,
 * so a device reset (cudaDeviceReset) after the first call is not supported.  All calls share the array and it keeps the last call's
 * partial sums (each call overwrites everything it reads, so nothing needs
 * clearing); calls that can overlap on the GPU race on it, so serialize them.
 */
vfl_status vfl_weight_grad_noalloc(const void* dpre, const void* x, int32_t rows, int32_t out, int32_t in,
                                   int32_t dtype, float* dW, float* db, void* stream);

/*
 * Roofline denominators of the fp32 kernels (measurement only; the paper has no counterpart): the
 * device's FP32 FMA throughput (VFL_PEAK_FFMA: eight independent FMA chains per thread) or its TF32
 * warp-MMA throughput (VFL_PEAK_TF32_MMA: eight independent m16n8k8 accumulators per warp), eight
 * 256-thread blocks per SM, `iters` iterations.  One warm-up launch, then one timed launch on the
 * legacy default stream of the current device: *flops its floating-point operations, *ms its
 * CUDA-event time.  Allocates and frees a small output buffer.  VFL_E_INVAL for an unknown kind or
 * iters < 1; the reason in vfl_last_error(NULL).
 */
#define VFL_PEAK_FFMA 0
#define VFL_PEAK_TF32_MMA 1
vfl_status vfl_measure_peak(int32_t kind, int64_t iters, double* flops, float* ms);

/* Last error message of the context (or of the last failed vfl_create / vfl_make_schedule when ctx is NULL);
 * error reporting has no counterpart in the paper. */
const char* vfl_last_error(const vfl_ctx* ctx);

#ifdef __cplusplus
}
#endif

#endif /* VFL_H */
