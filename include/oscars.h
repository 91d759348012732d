/*
 * oscars.h - C ABI of the GB300 (sm_103a) Oscars hot path.
 *
 * Oscars (arXiv 2102.08550) is semi-synchronous local SGD against a parameter
 * server: N workers with steady but different iteration times t_i^iter each
 * run tau_i local SGD steps between global barriers, where the barrier T* and
 * tau_i = floor(T* / t_i^iter) come from the paper's load-balance search
 * (Algorithm 1; Eq. 1-3); at the barrier the server merges the workers'
 * models (Eq. 4, first branch) and the workers pull the result.  This library
 * simulates the W workers and the server on ONE GPU: worker replicas, the
 * global model and all activations live in HBM, the workers' compute runs as
 * grouped kernels, and push / pull are stream-ordered buffer reads.
 *
 * Conventions for every entry point:
 *  - Status: every call returns an oscars_status; nothing throws or aborts
 *    across this boundary.  On failure the context (if any) keeps a message
 *    for oscars_last_error().
 *  - Pointers: "device" pointers are CUDA global-memory addresses of the
 *    current device; "host" pointers are ordinary process memory.  Where a
 *    parameter says "host or device" the library copies with
 *    cudaMemcpyDefault (unified addressing).
 *  - Ownership: the library never frees caller memory.  Caller buffers passed
 *    to oscars_create are BORROWED for the context's lifetime and must stay
 *    valid and unchanged in size until oscars_destroy.  The library owns the
 *    global model, the worker replicas and all work buffers.
 *  - Streams: work is ordered on the cuda_stream given at creation (NULL =
 *    the legacy default stream).  Calls that return values in host memory
 *    (tau_out, loss_out, schedule queries, pull to host) synchronise that
 *    stream first.  A context is not thread-safe.
 *  - Flat parameter vector ("canonical layout"): for layers l = 0..L-1 with
 *    fan-in d_l = dims[l] and fan-out d_{l+1} = dims[l+1], the weight W_l is
 *    stored row-major [d_{l+1}][d_l] followed by the bias b_l [d_{l+1}];
 *    layers follow each other without padding.  P = sum_l d_{l+1}(d_l + 1).
 */
#ifndef OSCARS_H
#define OSCARS_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct oscars_ctx oscars_ctx; /* opaque, library-owned */

typedef enum {
  OSCARS_OK = 0,
  OSCARS_EINVAL = 1,   /* bad argument or configuration                         */
  OSCARS_ENOMEM = 2,   /* host or device allocation failed                      */
  OSCARS_ECUDA = 3,    /* a CUDA call failed; see oscars_last_error              */
  OSCARS_ESTATE = 4,   /* call out of protocol order                            */
  OSCARS_ETIMEOUT = 5, /* a kernel's bounded wait ran out and it returned early */
  OSCARS_ENOTSUP = 6   /* valid request this build does not implement           */
} oscars_status;

typedef enum {
  OSCARS_MODEL_FLAT = 0, /* merge only: dims[0] = P parameters, no local steps */
  OSCARS_MODEL_MLP = 1,  /* ReLU MLP / softmax regression with softmax CE      */
  OSCARS_MODEL_CNN = 2   /* residual CNN on images (see below)                  */
} oscars_model;

/*
 * OSCARS_MODEL_CNN: the convolutional worker, a residual network of the kind
 * the paper trains (ResNet on CIFAR-10, Section "Dataset and DL Models") on
 * H x W x Cin NHWC images:
 *   s = relu(conv(x) + b0); per block u = relu(conv(h) + b_a),
 *   v = relu(conv(u) + b_b + h); g = mean over positions of v;
 *   logits = g W_f^T + b_f, softmax cross-entropy.
 * Convolutions are 3x3, stride 1, zero padding 1.  dims = {H, W, Cin, C, K}
 * (C channels, K classes), num_layers = number of residual blocks.  This
 * build supports H = W = 32, C = 64, 1 <= Cin <= 64, 2 <= K <= 32, 1 to 4
 * blocks, bf16 GEMMs, and a batch that is a multiple of 16 up to 256.
 * Canonical parameter layout: W_0 [C][3][3][Cin], b_0 [C], then per block
 * W_a [C][3][3][C], b_a, W_b, b_b, then W_f [K][C], b_f [K].  A shard holds
 * n images of H*W*Cin fp32 values (NHWC) and n labels.
 */

typedef enum {
  OSCARS_W_UNIFORM = 0,    /* w_k = 1/N: the average of Eq. 4 (first branch)        */
  OSCARS_W_LOCALSTEPS = 1, /* w_k = tau_k / sum_j tau_j: NOT in the paper            */
  OSCARS_W_EXPLICIT = 2    /* w_k given to every oscars_push_merge call              */
} oscars_weight_rule;

typedef enum {
  OSCARS_SEARCH_CAPPED = 0, /* Algorithm 1, also stopping once T > M * max(t)  */
  OSCARS_SEARCH_LITERAL = 1 /* Algorithm 1 as printed; needs min(t) < max(t)   */
} oscars_search_mode;

typedef enum {
  OSCARS_POLICY_OSCARS = 0,    /* tau_i from Algorithm 1 (load-balanced rounds)      */
  OSCARS_POLICY_BSP = 1,       /* tau_i = 1: a barrier after every iteration         */
  OSCARS_POLICY_LOCAL_SGD = 2  /* tau_i = I: average every I iterations (Motivation)  */
} oscars_policy;

typedef struct {
  int32_t num_workers;  /* N = W >= 1 (notation table); <= 256, MLP <= 64       */
  int32_t model;        /* oscars_model                                          */
  int32_t num_layers;   /* L >= 1 (MLP); 1 for FLAT                              */
  const int32_t* dims;  /* host, L+1 entries: input, hidden..., classes.  FLAT:  */
                        /* dims[0] = P.  MLP: classes <= 32                      */
  int32_t batch;        /* B, mini-batch rows per local step (MLP); fp32        */
                        /* softmax regression: 1..512, bf16 MLP: multiple of 32 */
                        /* up to 256                                            */
  float lr;             /* eta of Eq. 4                                          */
  float server_lr;      /* eta_s of the delta-form merge; 1.0 = Eq. 4's average  */
  int32_t weight_rule;  /* oscars_weight_rule                                    */
  int32_t bf16_gemm;    /* 1: GEMM operands rounded to bf16, fp32 accumulate;    */
                        /* 0: fp32 operands (only L = 1 supported)               */
  const double* speed;  /* host, W speed factors s_i > 0 (larger = faster), or   */
                        /* NULL when t_ticks is given                            */
  const int64_t* t_ticks;  /* host, W iteration times t_i^iter in ticks >= 1;   */
                           /* overrides speed when non-NULL                      */
  int64_t ticks_per_unit;  /* Q: t_i = max(1, floor(Q / s_i + 0.5)); 0 = 1000   */
  int64_t M;               /* local-step spread bound of Eq. 3, >= 1            */
  int32_t search_mode;     /* oscars_search_mode                                */
  const float* const* shard_x;   /* host array of W device-accessible pointers,  */
                                 /* worker i's samples [shard_n[i]][dims[0]] fp32 */
                                 /* row-major (bf16 MLP: 16-byte aligned).  Pinned */
                                 /* host memory is accepted: each round's rows are */
                                 /* then read over the host link by the kernels.   */
  const int32_t* const* shard_y; /* host array of W device-accessible pointers,  */
                                 /* [shard_n[i]] in [0, classes)                  */
  const int64_t* shard_n;        /* host, W shard sizes >= 1                      */
  const float* init_params;      /* host or device, P fp32 canonical layout,     */
                                 /* copied at creation; NULL = zeros (FLAT only)  */
  void* cuda_stream;             /* cudaStream_t, borrowed; NULL = default stream */
  int32_t flags;                 /* bit 0: launch each kernel of a round directly */
                                 /* instead of replaying a captured CUDA graph;   */
                                 /* bit 1: time every launch with CUDA events     */
                                 /* (graph mode: event nodes in the graph; see    */
                                 /* oscars_profile_read);                         */
                                 /* bit 2: run the workers of a round as up to 16 */
                                 /* concurrent branches (streams) instead of one  */
                                 /* launch per layer over all active workers;     */
                                 /* bit 3: do not use the one-launch round of a   */
                                 /* 2-layer MLP (per-layer kernels instead);      */
                                 /* bit 4: stamp the phases of that one-launch    */
                                 /* round (see oscars_phase_times)                */
} oscars_config;

/*
 * oscars_create - validate cfg, compute the schedule, allocate the model.
 *
 * Schedule (host): t_i^iter from speed (or t_ticks), then Algorithm 1 for the
 * barrier T* (Eq. 3 with its constraint; the search evaluates T = max(t)
 * first, keeps the first T with the smallest max_i mod(T, t_i) of Eq. 2) and
 * tau_i = floor(T* / t_i^iter) (the sentence after Eq. 3).
 * Memory: the global model and W replicas (fp32 master plus bf16 operand
 * copies in MLP/bf16 mode) and all per-step activations.  The shard pointers
 * are borrowed.  *out is set only on success.
 * Errors: EINVAL (bad sizes, NULL pointers, W out of range, t_i < 1, M < 1,
 * literal search with all t_i equal), ENOTSUP (a model shape outside what the
 * kernels handle), ENOMEM, ECUDA.
 */
oscars_status oscars_create(const oscars_config* cfg, oscars_ctx** out);

/* oscars_destroy - free everything the context owns.  NULL-safe.  Synchronises
 * the context's stream first. */
oscars_status oscars_destroy(oscars_ctx* ctx);

/*
 * oscars_local_steps - one round of worker compute (Eq. 4, "otherwise" branch).
 *
 * Every worker i starts from the current global model (the pull of the
 * parameter-server description, fused into its first step: nothing is copied)
 * and runs tau_i SGD steps x <- x - lr * g(x), each on the next B samples of
 * its own shard (a cursor per worker that persists across rounds and wraps
 * modulo shard_n[i]).  The results stay in the worker replicas, which are the
 * pushed models.  The simulated clocks advance by tau_i * t_i of compute and
 * mod(T*, t_i) of idle time (Eq. 1); synchronisation costs nothing.
 * tau_out: host, W int32 or NULL.  loss_out: host, W floats or NULL: worker
 * i's mean mini-batch loss over its tau_i steps.  Either being non-NULL
 * synchronises the stream.
 * Errors: ESTATE in FLAT mode or when the previous round was not merged yet;
 * ETIMEOUT if a kernel's bounded wait ran out; ECUDA.
 */
oscars_status oscars_local_steps(oscars_ctx* ctx, int32_t* tau_out, float* loss_out);

/*
 * oscars_losses_async - enqueue a copy of the per-worker mean mini-batch
 * losses of the last oscars_local_steps (W floats) into dst (host or device)
 * on the context's stream, without synchronising: the values are in dst once
 * the stream has reached this point (use pinned host memory for an
 * asynchronous copy).  Lets a training loop read each round's losses while
 * the next round runs.  Errors: EINVAL (NULL), ESTATE (no local steps yet, or
 * FLAT mode), ECUDA.
 */
oscars_status oscars_losses_async(oscars_ctx* ctx, float* dst);

/*
 * oscars_push_merge - server merge and global update (Eq. 4, first branch).
 *
 * x_g <- x_g + server_lr * sum_k w_k * delta_k, accumulated in fp32 registers
 * in worker order.  With deltas == NULL, delta_k = x^k - x_g from the worker
 * replicas of the last oscars_local_steps (MLP mode only); otherwise deltas
 * is a host array of W device pointers, each to P fp32 values in canonical
 * layout (any alignment).  w_k follows the weight rule; for OSCARS_W_EXPLICIT
 * `weights` is a host array of W floats (ignored otherwise, may be NULL).
 * Errors: ESTATE (deltas == NULL without pending local steps, or in FLAT
 * mode), EINVAL (NULL delta pointer, NULL weights for the explicit rule),
 * ECUDA.
 */
oscars_status oscars_push_merge(oscars_ctx* ctx, const float* const* deltas, const float* weights);

/*
 * oscars_pull - serve the global model.
 * dst != NULL: copy x_g (P fp32, canonical layout) into dst (host or device;
 * a host dst synchronises).  dst == NULL: write x_g into every worker replica
 * (an explicit pull; oscars_local_steps does not need it).
 */
oscars_status oscars_pull(oscars_ctx* ctx, float* dst);

/*
 * oscars_get_schedule - the schedule and simulated clocks.  Every output is a
 * host pointer and may be NULL.  T_star, max_wait: scalars (Eq. 3, Eq. 2 at
 * T*).  t_iter[W] ticks; tau[W]; wait[W] = mod(T*, t_i) (Eq. 1); clock[W] and
 * idle[W]: total simulated ticks and idle ticks so far.
 */
oscars_status oscars_get_schedule(const oscars_ctx* ctx, int64_t* T_star, int64_t* max_wait,
                                  int64_t* t_iter, int32_t* tau, int64_t* wait,
                                  int64_t* clock, int64_t* idle);

/*
 * oscars_set_local_steps - replace tau (host, W int32 >= 1), e.g. tau = 1 for
 * BSP or a fixed I for plain local SGD (the comparison schemes of the
 * paper's Motivation).  The barrier used by the simulated clock becomes
 * max_i tau_i * t_i.  Errors: EINVAL, ESTATE while a round is pending.
 */
oscars_status oscars_set_local_steps(oscars_ctx* ctx, const int32_t* tau);

/*
 * oscars_set_iteration_ticks - new iteration times t_iter[W] (host, ticks
 * >= 1), e.g. measured ones when worker speeds drift (the volatile cloud of
 * the paper's Introduction; the method itself assumes steady speeds, Section
 * "Problem Formulation").  Re-runs Algorithm 1 with the context's M and
 * search mode and replaces tau and the barrier T* for the following rounds;
 * the simulated clocks keep what they have accumulated.  Errors: EINVAL
 * (those of oscars_schedule_solve; the context is unchanged), ESTATE while a
 * round is pending.
 */
oscars_status oscars_set_iteration_ticks(oscars_ctx* ctx, const int64_t* t_iter);

/*
 * oscars_eval_loss - mean softmax cross-entropy of the global model on n
 * samples x [n][dims[0]] fp32 and labels y [n] (both device pointers), with
 * the same operand precision as training.  MLP mode; n >= 1; *loss is host.
 */
oscars_status oscars_eval_loss(oscars_ctx* ctx, const float* x, const int32_t* y, int64_t n,
                               float* loss);

/* One round of oscars_train. */
typedef struct {
  int64_t ticks;       /* simulated time at the end of the round: max_i clock_i   */
  int64_t barrier;     /* length of this round in ticks                          */
  float eval_loss;     /* eval loss of the merged global model (NaN without eval) */
  float worker_loss;   /* mean over workers of their mean mini-batch loss         */
} oscars_round_log;

/*
 * oscars_train - run up to `rounds` rounds natively: oscars_local_steps,
 * oscars_push_merge from the replicas (weights of the context's rule; the
 * explicit rule is refused), and, with eval_x != NULL, oscars_eval_loss of
 * the merged model on eval_x [eval_n][dims[0]] / eval_y [eval_n] (device).
 * With eval and target_loss > 0 it stops after the first round whose eval
 * loss is <= target_loss (the time-to-loss of the paper's convergence
 * comparison).  log: host array of `rounds` entries or NULL; rounds_done
 * (host, may be NULL) receives the number of rounds run.  With eval_x it
 * synchronises every round (it reads the losses and the eval loss).  Without
 * eval_x the rounds are pipelined one deep: round r, with an asynchronous
 * copy of its W losses into a pinned host slot, is enqueued before the host
 * waits for round r - 1 and reads that round's losses; the call returns after
 * the last round's losses were read.  Errors: those of the calls it makes;
 * EINVAL for rounds < 1 or eval_n < 1 with eval_x set; ETIMEOUT when a
 * kernel's bounded wait ran out in any round (without eval_x, reported after
 * the last round).
 */
oscars_status oscars_train(oscars_ctx* ctx, int32_t rounds, const float* eval_x, const int32_t* eval_y,
                           int64_t eval_n, float target_loss, oscars_round_log* log,
                           int32_t* rounds_done);

/*
 * oscars_read_replica - copy worker k's current model (the model it pushes at
 * the barrier; Section "Introduction": each worker holds a model copy) in
 * canonical layout into dst (host or device, P fp32).  MLP mode, 0 <= k < W.
 */
oscars_status oscars_read_replica(oscars_ctx* ctx, int32_t k, float* dst);

/*
 * oscars_profile_read - per-kernel-class device time of the launches made
 * since the last reset while flag bit 1 was set (CUDA events around every
 * launch on its stream; in graph mode they are event nodes of the captured
 * graph, so the times exclude host launch gaps).  Synchronises on the last
 * recorded event.  Fills up to `cap` entries: names[i] (library-owned, valid
 * until the next reset or destroy), ms_total[i], launches[i] (each may be
 * NULL).  Returns the number of classes, or -1 for a NULL ctx.
 * oscars_profile_reset clears the totals.
 */
int32_t oscars_profile_read(oscars_ctx* ctx, int32_t cap, const char** names, double* ms_total,
                            int32_t* launches);
oscars_status oscars_profile_reset(oscars_ctx* ctx);

/*
 * oscars_phase_times - with flag bit 4, the device time (microseconds, from
 * %globaltimer) of the three phases of every local step of worker 0 in the
 * last one-launch round of a 2-layer MLP: forward, last layer, weight
 * gradient + update, in that order (host us[3 * step + phase], up to cap).
 * Returns the number of values written, 0 without stamps, -1 on error.
 */
int32_t oscars_phase_times(oscars_ctx* ctx, int32_t cap, double* us);

/*
 * oscars_check_padding - look for writes where no kernel should write, in
 * place of a memory checker: the layout pads each weight and bias of a slot
 * to 64 elements, and that padding must stay zero in the fp32 slab and in
 * its bf16 copy; 256 guard words after each of the two hold a byte pattern
 * written at creation.  *bad (host) receives the number of padding values
 * that are not zero (MLP mode) plus the guard words that changed (MLP and
 * CNN).  Synchronises the stream and copies both slabs to the host: meant
 * for tests and debugging, not for a training loop.  Not a step of the
 * method.  Errors: EINVAL (NULL), ESTATE (FLAT mode), ENOMEM, ECUDA.
 */
oscars_status oscars_check_padding(oscars_ctx* ctx, int64_t* bad);

/*
 * oscars_debug_slab - the device address of the context's fp32 slab and its
 * slot stride in floats (slot k < W is worker k's replica, slot W the global
 * model; each tensor starts on a 64-element boundary), for tests of the
 * layout.  Writing through it changes the model.  Errors: EINVAL (NULL).
 */
oscars_status oscars_debug_slab(const oscars_ctx* ctx, float** slab, int64_t* slot_stride);

/*
 * oscars_check_wait_timeout - exercise the failure path of the kernels'
 * bounded waits.  Every wait of a kernel in this library on an mbarrier (a
 * TMA stage, a tensor-core accumulator, a peer CTA's data) gives up after a
 * fixed number of polls, records a code in the context's device error word
 * and lets the kernel end, and the next call that reads results reports
 * OSCARS_ETIMEOUT.  This call runs that path on purpose: one GPU thread waits
 * `polls` polls (1 .. 2^20) on an mbarrier that nothing completes, on the
 * context's stream, then the host reads and clears the error word as after a
 * round.  It returns OSCARS_ETIMEOUT when the path works; the context stays
 * usable.  Not a step of the method (the paper assumes steady workers and
 * has no failure model).  Errors: EINVAL (NULL, polls out of range), ESTATE
 * (FLAT mode: no kernel error word), ECUDA.
 */
oscars_status oscars_check_wait_timeout(oscars_ctx* ctx, int32_t polls);

/* oscars_num_params - P of the context (canonical layout). */
oscars_status oscars_num_params(const oscars_ctx* ctx, int64_t* P);

/* Message of the last failure on ctx ("" if none).  Valid until the next call. */
const char* oscars_last_error(const oscars_ctx* ctx);

/* Name of a status code. */
const char* oscars_status_string(int32_t status);

/*
 * Host-only helpers (no GPU needed): the scheduler of oscars_create.
 *
 * oscars_iteration_ticks: t[i] = max(1, floor(Q / speed[i] + 0.5)) in fp64,
 * then int64 (Q = ticks_per_unit, 0 = 1000); speed[i] > 0.
 * oscars_schedule_solve: Algorithm 1 on t_iter[n] with bound M and the given
 * search mode; outputs T*, the max wait at T* (Eq. 2) and tau[n]
 * (all host, tau may be NULL).  Errors: EINVAL.
 * oscars_merge_weights: the fp32 weights of a rule for local-step counts
 * tau[n] (uniform or local-steps), computed in fp64 and rounded once.
 */
oscars_status oscars_iteration_ticks(const double* speed, int32_t n, int64_t ticks_per_unit,
                                     int64_t* t_iter);
oscars_status oscars_schedule_solve(const int64_t* t_iter, int32_t n, int64_t M,
                                    int32_t search_mode, int64_t* T_star, int64_t* max_wait,
                                    int32_t* tau);
oscars_status oscars_merge_weights(int32_t rule, const int32_t* tau, int32_t n, float* w);

/*
 * oscars_policy_local_steps - the local-step counts of one round under a
 * synchronisation scheme (oscars_policy): Algorithm 1 (with M and the search
 * mode), BSP (tau_i = 1) or local SGD with period I (tau_i = I, I >= 1; the
 * scheme of the paper's Motivation, where the fast workers wait for the
 * slowest).  tau[n] (host) receives the counts and *barrier (host, may be
 * NULL) the round length max_i tau_i * t_i, which equals T* for Algorithm 1.
 * Feed tau to oscars_set_local_steps to run a context under the scheme.
 * Errors: EINVAL (unknown policy, I < 1, or the errors of
 * oscars_schedule_solve).
 */
oscars_status oscars_policy_local_steps(int32_t policy, const int64_t* t_iter, int32_t n, int64_t M,
                                        int32_t search_mode, int32_t I, int32_t* tau, int64_t* barrier);

/*
 * oscars_partition_sizes - data-partition load balancing (the paper names the
 * subsection and leaves it empty; this is the library's reading): split a
 * data set of `total` samples into n contiguous shards whose sizes follow the
 * per-round consumption of the workers, so that every worker sweeps its shard
 * in the same number of rounds and every sample is visited equally often.
 * weight[n] (host, >= 1) are the proportions, normally tau (samples per round
 * = tau_i * B).  The data set is handed out in whole units of `unit` samples
 * (normally B): Q = floor(total / unit) units in proportion to the weights
 * by largest remainder (Hamilton's apportionment; exact integer arithmetic,
 * ties to the lower index); sizes[n] (host) receive samples, a multiple of
 * unit each, summing to Q * unit.  sizes is written only on success.
 * Errors: EINVAL (NULL, n < 1, unit < 1, a weight < 1, or a worker that
 * would get no unit).
 */
oscars_status oscars_partition_sizes(const int64_t* weight, int32_t n, int64_t total, int64_t unit,
                                     int64_t* sizes);

/*
 * oscars_round_clusters - the worker lists of the one-launch round kernel
 * (one thread-block cluster per worker, the worker's model on chip; Eq. 4,
 * "otherwise" branch) when fewer of its clusters fit on the device than there
 * are workers.  tau[n] (host, >= 1): the local steps of each worker this
 * round; max_clusters: the clusters that fit at once (<= 0 or >= n: one
 * cluster per worker).  Workers by decreasing tau (ties by index) go, one at
 * a time, to the cluster with the least work so far (ties to the lower
 * cluster), a worker costing tau + 1/2 (its steps and about half a step of
 * model load): longest processing time first.  order[n] (host) receives the
 * workers cluster by cluster, first[] (host, room for n + 1) the start of
 * each cluster's run in order plus the end, *clusters their number; a
 * cluster runs its workers one after the other.  Errors: EINVAL (NULL,
 * n < 1, a tau < 1).
 */
oscars_status oscars_round_clusters(const int32_t* tau, int32_t n, int32_t max_clusters, int32_t* order,
                                    int32_t* first, int32_t* clusters);

/*
 * oscars_merge - the server update of Eq. 4 (first branch) on caller buffers,
 * without a context: x_g[p] <- x_g[p] + server_lr * sum_k w[k] * deltas[k][p]
 * for p < P.  x_g: device, P fp32, updated in place.  deltas: host array of W
 * device pointers to P fp32 each.  w: host, W floats.  Any alignment;
 * 16-byte aligned pointers take the vector path.  Ordered on `stream`
 * (cudaStream_t or NULL).  W <= 256.  Errors: EINVAL, ECUDA.
 */
oscars_status oscars_merge(float* x_g, const float* const* deltas, const float* w, int32_t W,
                           int64_t P, float server_lr, void* stream);

/*
 * oscars_gemm_bf16_nt - C[M][N] = sum_k A[m][k] * B[n][k] on the tcgen05
 * tensor cores, the contraction of the workers' dense layers (Eq. 4,
 * "otherwise" branch: forward and backward products) without a fused
 * epilogue.  A: device, [M][K] bf16 row-major; B: device, [N][K] bf16
 * row-major; both 16-byte aligned.  C: device, [M][N] fp32 row-major,
 * overwritten.  M a multiple of 128, K a multiple of 8, N >= 1.  fp32
 * accumulation.  Ordered on `stream`.  Errors: EINVAL, ECUDA.
 */
oscars_status oscars_gemm_bf16_nt(const void* A, const void* B, float* C, int32_t M, int32_t N, int32_t K,
                                  void* stream);

/*
 * oscars_softreg_steps_noalloc - one worker's tau local SGD steps of fp32
 * softmax regression, like one worker of oscars_local_steps, for callers that
 * cannot allocate device memory when they call: code recording a CUDA graph
 * in global capture mode (where cudaMalloc is refused), hosts whose memory
 * pool owns the whole GPU, and loops that cannot pay for cudaMalloc/cudaFree,
 * which may synchronise the device.  The paper has no counterpart; this is a
 * deployment convenience.  It allocates nothing: its scratch (argument tables
 * and per-step loss partials) is a fixed 64 KB array inside the library that
 * every GPU which loads the library keeps until the process exits.
 *
 * params_in / params_out: device, classes*dim + classes fp32 each, canonical
 * layout (W [classes][dim], then b [classes]); they may be the same buffer.
 * x: device [n][dim] fp32 (any alignment; with dim % 4 == 0 and x 16-byte
 * aligned the rows are read as 16-byte vectors); y: device [n] int32 labels
 * in [0, classes).  Step s uses rows (cursor + s*batch + b) mod n, b < batch.
 * loss_out: device, 1 float: the mean mini-batch loss over the tau steps.
 * Ordered on `stream`.  1 <= tau <= 16320 (the scratch holds one loss
 * partial per step); larger tau, classes outside [2, 32] or bad pointers give
 * EINVAL; batch > 512, or shapes whose weights plus one batch exceed shared
 * memory, ENOTSUP.
 * The first call on a device looks up the scratch address (once per device);
 * make that first call before any stream capture.  Every call shares the one
 * scratch array and leaves its contents behind; each call writes all it reads
 * first, so nothing needs clearing, but calls that overlap on the GPU (other
 * streams, other threads) race on it.
 */
oscars_status oscars_softreg_steps_noalloc(const float* params_in, float* params_out, const float* x,
                                           const int32_t* y, int64_t n, int64_t cursor, int32_t tau,
                                           int32_t dim, int32_t classes, int32_t batch, float lr,
                                           float* loss_out, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* OSCARS_H */
