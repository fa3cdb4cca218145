/* lsgd.h -- C ABI of the GB300 local / post-local SGD hot path.
 *
 * Method: "Don't Use Large Mini-Batches, Use Local SGD" (Lin, Stich, Patel, Jaggi).  K workers
 * are simulated on one GPU as K model replicas held in one replica-major buffer.  One local step
 * (Eq. 2, left part; the inner loop of Algorithm 1) samples each worker's mini-batch from its own
 * shard, runs forward/backward per replica and applies a local momentum-SGD update; a round ends
 * with the K-way model average (Eq. 2, right part).  Post-local SGD (Sec. 3, Algorithm 2) averages
 * after every step before the switch step t' and every H steps after it.
 *
 * Conventions (every entry point):
 *  - Returns an lsgd_status; on error, out-parameters are left untouched and lsgd_last_error()
 *    describes the failure.  A failed call leaves the context usable unless it returns LSGD_ECUDA.
 *  - The library owns every device buffer it allocates (through the caller's allocator if one is
 *    given); the caller owns every buffer it passes in, and the library copies what it keeps.
 *  - Step calls are asynchronous on the stream given at creation; calls that return host data
 *    synchronise that stream first.  A context is not thread-safe: one host thread at a time.
 *  - Parameter vectors use the canonical packed order: for each dense layer l = 1..L, W_l row-major
 *    [out_l][in_l] then b_l [out_l]; for ResNet-20, per convolution (stem first) its weight
 *    [Cout][3][3][Cin], BN gamma [Cout], BN beta [Cout], then the classifier W [classes][4 base]
 *    and b [classes].  Internally each tensor is padded to 256-byte alignment.
 *  - Dataset rows are fp32, HWC for images; labels are int32 class ids, targets fp32.
 */
#ifndef LSGD_H
#define LSGD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define LSGD_MAX_LAYERS 8
#define LSGD_MAX_MILESTONES 4

typedef enum {
  LSGD_OK = 0,
  LSGD_EINVAL = 1,       /* bad argument or configuration */
  LSGD_ENOMEM = 2,       /* allocation failed (the context stays valid) */
  LSGD_ECUDA = 3,        /* a CUDA call failed; the context should be destroyed */
  LSGD_ESTATE = 4,       /* call out of order (e.g. a step before lsgd_set_dataset) */
  LSGD_ENONFINITE = 5,   /* lsgd_check_finite found a NaN or Inf */
  LSGD_ETIMEOUT = 6,     /* a bounded device-side wait ran out */
  LSGD_EUNSUPPORTED = 7, /* valid but not supported by this build (e.g. shape limits) */
  LSGD_EIO = 8           /* checkpoint file error */
} lsgd_status;

typedef enum {
  LSGD_MLP = 0,      /* dense ReLU network with softmax cross-entropy; 1 layer = softmax regression */
  LSGD_LSQ = 1,      /* least squares f_i(w) = 1/2 (a_i^T w - t_i)^2, one layer, no bias */
  LSGD_RESNET20 = 2  /* CIFAR ResNet-20 (He et al. 2016) with option-A shortcuts */
} lsgd_model_kind;

typedef enum { LSGD_FP32 = 0, LSGD_BF16 = 1 } lsgd_precision;
typedef enum { LSGD_INIT_ZERO = 0, LSGD_INIT_HE = 1 } lsgd_init_kind;

typedef struct {
  lsgd_model_kind kind;
  int n_layers;                         /* dense layers (MLP, LSQ) */
  int widths[LSGD_MAX_LAYERS + 1];      /* widths[0] = input dim ... widths[n_layers] = outputs */
  int init;                             /* lsgd_init_kind: He-normal (fan-in) or zeros */
  int in_h, in_w, in_c;                 /* ResNet: image geometry (32, 32, 3) */
  int n_classes, base_ch, res_blocks;   /* ResNet: 10, 16, 3 */
} lsgd_model;

/* gamma(s), Sec. A.3 / A.4: eta_hat = K eta if scale_by_K; linear warm-up from eta adding
 * (eta_hat - eta) / (warmup_epochs N / (K B)) per step, capped at eta_hat; then gamma is
 * multiplied by `decay` at every step s >= floor(milestone_frac[i] * T). */
typedef struct {
  double base_lr;
  int scale_by_K;
  double warmup_epochs;
  int n_milestones;
  double milestone_frac[LSGD_MAX_MILESTONES];
  double decay;
} lsgd_lr_schedule;

/* Optional device allocator (NULL: cudaMallocAsync / cudaFreeAsync on the context's stream).
 * alloc returns a device pointer aligned to at least 256 bytes, or NULL on failure. */
typedef struct {
  void* (*alloc)(void* user, size_t bytes, void* stream);
  void (*free)(void* user, void* ptr, void* stream);
  void* user;
} lsgd_allocator;

typedef struct {
  int K;                 /* workers (replicas), >= 1 */
  int B_loc;             /* local mini-batch size, >= 1 */
  int H;                 /* local steps per averaging round after the switch, >= 1 */
  int64_t t_switch;      /* post-local switch step t' (H = 1 for steps s < t'); < 0: plain local SGD */
  int64_t total_steps;   /* T; 0 derives T = ceil(epochs N / (K B)) */
  double epochs;
  int64_t N;             /* dataset rows that lsgd_set_dataset will provide; >= K */
  lsgd_model model;
  lsgd_lr_schedule lr;
  double momentum;       /* m; 0 = plain SGD */
  int nesterov;
  double weight_decay;   /* lambda; never applied to BatchNorm gamma / beta */
  uint64_t seed;         /* keys Philox4x32-10 for sampling and initialisation */
  int precision;         /* lsgd_precision: FP32 = fp32 everywhere; BF16 = bf16 GEMM operands,
                            fp32 accumulation, fp32 master weights and optimizer state */
  int fused_update;      /* BF16 dense models on tcgen05: 1 = the weight-gradient epilogue (and the
                            bias-gradient sum) apply the local update directly, so the gradient is
                            never written to memory; bit-identical to 0, which runs the stand-alone
                            update kernel over the whole K x d buffer.  Ignored elsewhere. */
  int hier_block;        /* hierarchical local SGD (Sec. D): > 0 = after every H-step round the
                            hier_block consecutive replicas of each block are averaged, and every
                            hier_rounds-th round (and the run's last step) all K; must divide K.
                            0 = off.  The mini-batch phase of post-local SGD averages globally. */
  int hier_rounds;       /* H^b >= 1 */
  int compress;          /* lsgd_compress: averaging of compressed model differences (Sec. B.3)
                            relative to the round-start model w_ref.  Not with hier_block;
                            K <= 1024. */
  double global_momentum;/* m_g > 0: global momentum at every average (Sec. C.3.1):
                            u_g = m_g u_g + (w_ref - mean_k w^k) / gamma, w_ref -= gamma u_g.
                            Not with compress or hier_block. */
  int h_warmup;          /* lsgd_h_warmup: local-step warm-up (Sec. C; Sec. 4's ImageNet runs).  The
                            round starting at step s0 in epoch e = floor(s0 K B_loc / N) <
                            h_warmup_epochs = P has 1 + floor((H-1) e / P) steps (LINEAR),
                            min(H, 2^floor(e log2(H) / P)) (EXPONENTIAL) or 1 (CONSTANT); H from
                            epoch P on.  Replaces the post-local switch (t_switch must be < 0);
                            not with hier_block. */
  double h_warmup_epochs;
  int sampling;          /* lsgd_sampling */
} lsgd_config;

typedef enum {
  LSGD_HWARM_NONE = 0,
  LSGD_HWARM_LINEAR = 1,
  LSGD_HWARM_EXPONENTIAL = 2,
  LSGD_HWARM_CONSTANT = 3
} lsgd_h_warmup;

typedef enum {
  LSGD_SAMPLE_SHARDS = 0,    /* static contiguous shards of S = floor(N/K) points, B uniform draws
                                with replacement per step: k S + mulhi(Philox word, S) */
  LSGD_SAMPLE_RESHUFFLE = 1  /* Sec. 4 / A.4: the data is re-permuted globally every epoch and
                                partitioned disjointly; worker k's t-th step of epoch e takes
                                pi_e(k S + (t B + j) mod S), j < B, where pi_e is a four-round
                                Feistel permutation of [0, N) keyed by Philox (seed, e) with cycle
                                walking; N < 2^31 */
} lsgd_sampling;

typedef enum {
  LSGD_COMPRESS_NONE = 0,
  LSGD_COMPRESS_SIGN = 1,    /* Algorithm 4: local steps w -= gamma sign(step); the average becomes
                                w_ref -= (1/K) sum_k sign(Delta_k) ||Delta_k||_1 / d,
                                Delta_k = w_ref - w^k */
  LSGD_COMPRESS_EF_SIGN = 2  /* Algorithm 5: plain local steps; Delta_k = w_ref - w^k + e^k, the same
                                compressed average, and e^k = Delta_k - sign(Delta_k) ||Delta_k||_1 / d */
} lsgd_compress;

typedef struct lsgd_ctx lsgd_ctx;

/* Create a context: validates cfg, allocates the replica-major buffers (w, u, g fp32 and the bf16
 * shadow of w in BF16 mode, all [K][d_pad]), initialises w_(0) from cfg.seed and copies it to
 * every replica ("synchronize to have the same initial models", Algorithm 1).  `cuda_stream` is a
 * cudaStream_t (NULL = legacy default stream).  LSGD_EINVAL for K, B_loc, H < 1, N < K, bad model
 * widths; LSGD_EUNSUPPORTED for BF16 dense layers whose input width is not a multiple of 8. */
lsgd_status lsgd_create(const lsgd_config* cfg, const lsgd_allocator* alloc, void* cuda_stream,
                        lsgd_ctx** out);
void lsgd_destroy(lsgd_ctx* ctx);

/* Copy the training set (host pointers, N rows of widths[0] fp32 and N int32 labels in
 * [0, classes)) to the device.  Worker k owns rows [k floor(N/K), (k+1) floor(N/K)) (the data is
 * "partitioned among the GPUs", Sec. A.4).  N must equal cfg.N.  LSQ uses lsgd_set_targets. */
lsgd_status lsgd_set_dataset(lsgd_ctx* ctx, const float* X, const int32_t* labels, int64_t N);
lsgd_status lsgd_set_targets(lsgd_ctx* ctx, const float* X, const float* targets, int64_t N);

/* One local step s on all K replicas (Eq. 2 left / Algorithm 1 inner loop): sample
 * I^k_s = k floor(N/K) + mulhi(Philox(ctr = (j/4, s, k, 0), key = seed)[j mod 4], floor(N/K)),
 * gather and cast the rows, forward, loss, backward, then the fused update
 * g' = g + lambda w; u = m u + g'; w -= gamma(s) (g' + m u | u | g').  Does not average. */
lsgd_status lsgd_local_step(lsgd_ctx* ctx);

/* Same step, but on a caller-supplied mini-batch x [K][B_loc][widths[0]] fp32 and labels
 * [K][B_loc] (or targets for LSQ), replica-major, instead of sampling the resident dataset.
 * `on_device` = 0: host pointers, copied into one of two library-owned staging buffers on a copy
 * stream of the library's (asynchronously from pinned memory, synchronously from pageable
 * memory), so that the copy of the next batch can run while this step computes; the step waits
 * for its copy, a copy waits until the step two batches earlier has read its buffer.  Either way
 * the caller keeps the buffers unchanged until the step has been reached (lsgd_losses,
 * lsgd_synchronize). */
lsgd_status lsgd_local_step_batch(lsgd_ctx* ctx, const float* x, const void* labels_or_targets,
                                  int on_device);

/* The K-way average w^k := (1/K) sum_k w^k for every k (Eq. 2 right; the all-reduce and model
 * update that close each round of Algorithm 1); momentum buffers stay local (Sec. A.4).
 * Refreshes the bf16 shadow.  With cfg.compress or cfg.global_momentum the average is the
 * corresponding variant (gamma of the step that ended the round) and the result also becomes the
 * next round's w_ref; lsgd_set_params(ctx, -1, ...) resets w_ref. */
lsgd_status lsgd_sync_average(lsgd_ctx* ctx);

/* Block average of hierarchical local SGD (Sec. D): every replica becomes the mean of the
 * hier_block replicas of its block.  LSGD_ESTATE if the context has no blocks. */
lsgd_status lsgd_block_average(lsgd_ctx* ctx);

/* n_steps local steps from the current step counter, averaging after every step s that ends a
 * round: s < t' (post-local first phase), (s + 1 - max(t', 0)) mod H == 0, or s == T - 1.  With
 * hier_block > 0 the r-th round end after the switch is a block average unless r is a multiple
 * of hier_rounds (or s == T - 1).  With the fused update (bf16 dense models) and plain averaging,
 * a step that ends with the global average forms it inside its own update launches: each weight
 * tile is taken through all K replicas, updated per replica as usual, and the mean of the updated
 * tiles goes to every replica (the same bits as the separate K-way average, without writing and
 * re-reading the per-replica models). */
lsgd_status lsgd_run(lsgd_ctx* ctx, int64_t n_steps);

/* One step of lsgd_run's schedule on a caller-supplied mini-batch (arguments as for
 * lsgd_local_step_batch): the local step, then the average the schedule puts at its end (global or
 * block), counted like lsgd_run's.  Where the step ends with the plain global average and the
 * update runs in the weight-gradient epilogue, the average is formed inside that step's update
 * launches (Eq. 2: the mean of the updated replicas, to the same bits as the separate average). */
lsgd_status lsgd_run_batch(lsgd_ctx* ctx, const float* x, const void* labels_or_targets,
                           int on_device);

/* Replica k's fp32 parameters (k = -1: the element-wise mean over replicas, computed in fp64 on
 * the host) in canonical order, n = lsgd_num_params() elements, to host or device memory. */
lsgd_status lsgd_params(lsgd_ctx* ctx, int k, float* dst, int dst_is_device, size_t n);
lsgd_status lsgd_momentum(lsgd_ctx* ctx, int k, float* dst, int dst_is_device, size_t n);
/* Overwrite replica k's parameters / momentum (k = -1: every replica) from host memory. */
lsgd_status lsgd_set_params(lsgd_ctx* ctx, int k, const float* src, size_t n);
lsgd_status lsgd_set_momentum(lsgd_ctx* ctx, int k, const float* src, size_t n);

typedef enum {
  LSGD_STATE_WREF = 0,            /* round-start model w_ref (k = 0) */
  LSGD_STATE_ERROR = 1,           /* error-feedback memory e^k of replica k (Algorithm 5) */
  LSGD_STATE_GLOBAL_MOMENTUM = 2  /* global momentum u_g (k = 0; Sec. C.3.1) */
} lsgd_sync_state_kind;
/* Read / overwrite the synchronisation state of the compressed and global-momentum averages, n =
 * lsgd_num_params() floats of host memory in canonical order.  k selects the replica for
 * LSGD_STATE_ERROR (k = -1 on write: every replica) and must be 0 for the others.  LSGD_ESTATE if
 * the configuration does not keep that state (w_ref exists with compress or global_momentum, e^k
 * with LSGD_COMPRESS_EF_SIGN, u_g with global_momentum). */
lsgd_status lsgd_sync_state(lsgd_ctx* ctx, int which, int k, float* dst, size_t n);
lsgd_status lsgd_set_sync_state(lsgd_ctx* ctx, int which, int k, const float* src, size_t n);

/* Per-replica mean mini-batch loss of the last `n_steps` steps, [n_steps][K] fp32, oldest first.
 * The history holds the last T steps. */
lsgd_status lsgd_losses(lsgd_ctx* ctx, float* dst, int64_t n_steps);
/* The same read, enqueued on the context's stream without waiting: dst (host memory the caller
 * owns; pinned for a truly asynchronous copy) holds the values once the stream has passed the
 * copy, e.g. after lsgd_synchronize. */
lsgd_status lsgd_losses_async(lsgd_ctx* ctx, float* dst, int64_t n_steps);
/* Wait until every step, copy and average enqueued on the context so far has completed. */
lsgd_status lsgd_synchronize(lsgd_ctx* ctx);

/* The mini-batch indices I^k_s of step s for every worker, [K][B_loc] int32 (host). */
lsgd_status lsgd_debug_indices(lsgd_ctx* ctx, int64_t step, int32_t* dst);

/* Mean loss of replica k (k = -1: replica 0 right after a sync) over the first n dataset rows,
 * computed with the same forward kernels (no update). */
lsgd_status lsgd_eval_loss(lsgd_ctx* ctx, int k, int64_t n, double* loss);

/* LSGD_ENONFINITE if any replica parameter is NaN or Inf (after lsgd_device_status's check). */
lsgd_status lsgd_check_finite(lsgd_ctx* ctx);

/* Failure detection for the device-side waits.  Every wait inside the tensor-core kernels (on a TMA
 * arrival, an MMA completion or a free pipeline stage) is bounded (about 2 s of SM clocks); when
 * one runs out the kernel records it in a device flag, stops issuing work, drains its copies in
 * flight, frees its tensor memory and exits, so the context stays usable.  lsgd_device_status
 * synchronises ctx's stream (ctx may be NULL), reads and clears that flag and returns
 * LSGD_ETIMEOUT if it was set (the results computed since the previous check are then invalid),
 * else LSGD_OK.  The flag is per device and process. */
lsgd_status lsgd_device_status(lsgd_ctx* ctx);

/* Exercises that expiry path on its own: one thread waits, through the kernels' bounded wait,
 * with a limit of limit_ms (0..1000) milliseconds, on an mbarrier phase that completes only if
 * arrive != 0.  Returns LSGD_OK when the phase completed, LSGD_ETIMEOUT when the wait ran out
 * (the device flag is consumed), on the current device and the given stream. */
lsgd_status lsgd_bounded_wait_selftest(int arrive, double limit_ms, void* stream);

/* Checkpoint / resume of w, u (all replicas), the synchronisation state (w_ref, e^k, u_g where the
 * configuration keeps it), the step and sync counters.  Philox is counter based so no generator
 * state is stored.  lsgd_load requires a context created with the same config. */
lsgd_status lsgd_save(lsgd_ctx* ctx, const char* path);
lsgd_status lsgd_load(lsgd_ctx* ctx, const char* path);

/* The schedule a context created from cfg follows, computed on the host without a GPU: for local
 * steps s = 0 .. n_steps-1, lr[s] = gamma(s) (Sec. A.3 warm-up, Sec. A.4 decays) and sync_kind[s] =
 * the average that ends step s (0 none, 1 block average, 2 global average: post-local switch,
 * local-step warm-up, hierarchical rounds).  Either array may be NULL.  Validates cfg exactly as
 * lsgd_create does. */
lsgd_status lsgd_schedule(const lsgd_config* cfg, int64_t n_steps, double* lr, int32_t* sync_kind);

int64_t lsgd_num_params(const lsgd_ctx* ctx);   /* d, canonical (unpadded) */
int64_t lsgd_step_count(const lsgd_ctx* ctx);   /* local steps taken so far (next step's s) */
/* Make s the next step's index, 0 <= s <= T: the learning rate, the round ends and the sampled
 * mini-batches follow s from there (s = 0 starts the schedule again from the current model).
 * Parameters, momentum, synchronisation state and the counters of syncs and launches are kept;
 * loss-history entries are overwritten as steps reuse their slots.  Steps already enqueued are
 * unaffected (each carries its own s). */
lsgd_status lsgd_set_step(lsgd_ctx* ctx, int64_t step);
int64_t lsgd_sync_count(const lsgd_ctx* ctx);   /* global averages performed so far */
int64_t lsgd_block_sync_count(const lsgd_ctx* ctx); /* block averages performed so far */
int64_t lsgd_total_steps(const lsgd_ctx* ctx);  /* T */
double lsgd_lr_at(const lsgd_ctx* ctx, int64_t step); /* gamma(s) as used by the update */
/* Kernel launches issued by this context since creation (for launch accounting). */
int64_t lsgd_kernel_launches(const lsgd_ctx* ctx);
/* Message for the last failed call on this context (or creation failure if ctx is NULL);
 * valid until the next call on the same context. */
const char* lsgd_last_error(const lsgd_ctx* ctx);

/* ---- Tracing: CUDA-event timing of each phase of the step on the context's stream ---- */
typedef enum {
  LSGD_PH_INPUT = 0,    /* index sampling + row gather / cast (or the caller batch's copy) */
  LSGD_PH_FORWARD = 1,  /* forward GEMMs / convolutions */
  LSGD_PH_LOSS = 2,     /* softmax cross-entropy (or least-squares) loss and its gradient */
  LSGD_PH_BACKWARD = 3, /* data / weight gradient products and bias sums (with fused_update: the
                           data-gradient products and the bias sum + update launches) */
  LSGD_PH_UPDATE = 4,   /* the local update kernel (with fused_update: the weight-gradient
                           launches that apply the update in their epilogue) */
  LSGD_PH_AVERAGE = 5,  /* the K-way average kernel */
  LSGD_NUM_PHASES = 6
} lsgd_phase;

typedef struct {
  int64_t count[LSGD_NUM_PHASES]; /* timed intervals per phase */
  double ms[LSGD_NUM_PHASES];     /* summed device time per phase (CUDA events) */
} lsgd_profile;

/* Start (enable = 1) or stop recording; enabling clears the accumulated times.  While enabled,
 * each phase of every step and average is bracketed by CUDA events on the context's stream. */
lsgd_status lsgd_profile_enable(lsgd_ctx* ctx, int enable);
/* Synchronise the stream and return the times accumulated since recording was enabled. */
lsgd_status lsgd_profile_read(lsgd_ctx* ctx, lsgd_profile* out);

/* ---- Stand-alone device kernels of the path (device pointers, asynchronous on `stream`) ---- */

/* K-way average of Eq. 2 (right) over replica-major W [K][d] fp32 (d a multiple of 4, W 16-byte
 * aligned): every replica's row becomes the fp32 mean; if Wb != NULL its bf16 copy is written to
 * Wb [K][d].  LSGD_EINVAL on bad sizes or alignment. */
lsgd_status lsgd_kway_average(float* W, uint16_t* Wb, int K, int64_t d, void* stream);

/* The fused local update of Sec. C.3.1 / A.4 over n elements (n a multiple of 4, 16-byte aligned
 * pointers): g' = g + (wd_mask ? lambda w : 0); u = m u + g'; w -= lr (nesterov ? g' + m u : u),
 * or w -= lr g' when m == 0 (u untouched, may be NULL); Wb (optional) receives bf16(w).  Elements
 * whose index modulo `period` is at least `decay_end` get no weight decay (period = 0: all do). */
lsgd_status lsgd_sgd_update(float* w, float* u, const float* g, uint16_t* Wb, int64_t n, float lr,
                            float momentum, int nesterov, float weight_decay, int64_t period,
                            int64_t decay_end, void* stream);

/* Grouped bf16 GEMM of the dense layers' products: C[g] = A[g] B[g]^T for g < G, with A[g] an
 * M x Kd matrix stored [M][Kd] (a_mn = 0, "K-major") or [Kd][M] (a_mn = 1), B[g] an N x Kd matrix
 * stored [N][Kd] (b_mn = 0) or [Kd][N] (b_mn = 1), groups packed back to back, C [G][M][N] fp32.
 * engine 0 = tcgen05 / TMEM / TMA kernel, 1 = SIMT kernel (fp32 accumulation in both).  The
 * contiguous extent of each operand must be a multiple of 8 elements and the pointers 16-byte
 * aligned (LSGD_EINVAL otherwise).  Device pointers, asynchronous on `stream`. */
lsgd_status lsgd_grouped_gemm_bf16(const uint16_t* A, int a_mn, const uint16_t* B, int b_mn, float* C,
                                   int M, int N, int Kd, int G, int engine, void* stream);

/* Per-worker BatchNorm batch statistics (Sec. A.4: each worker normalises with the statistics of
 * its own mini-batch): for y [G][P][C] fp32 (G replicas, P = batch x height x width positions, C
 * channels, channel fastest) writes mean[G][C] and rstd[G][C] = 1 / sqrt(biased variance + 1e-5).
 * Two deterministic passes: per-chunk mean and squared deviations, then Chan's pairwise
 * combination in chunk order.  The chunk partials live in a scratch buffer of
 * G x ceil(P / 1024) x C x 2 floats that this call allocates and frees on `stream` (stream-ordered
 * allocation).  Device pointers; 1 <= C <= 256, G <= 65535, P <= 65535 x 1024; LSGD_EINVAL
 * otherwise, LSGD_ENOMEM if the scratch cannot be allocated. */
lsgd_status lsgd_batchnorm_stats(const float* y, int64_t P, int C, int G, float* mean, float* rstd,
                                 void* stream);

/* Weight gradient of a 3x3 convolution with zero padding 1 and stride s (1 or 2), the product
 * behind ResNet-20's backward pass (Sec. A.2), for G independent groups on the tensor cores:
 *   dW[g][co][kh][kw][ci] = sum over b, oy, ox of dy[g][b][oy][ox][co] x[g][b][oy s + kh - 1][ox s + kw - 1][ci]
 * (x zero outside the image).  x [G][B][s Hout][s Wout][Cin] and dy [G][B][Hout][Wout][Cout] are
 * NHWC bf16 device arrays (16-byte aligned), dW [G][Cout][3][3][Cin] fp32 device, fully
 * overwritten.  The column matrix of every 64-pixel block is built in shared memory; one fp32
 * partial per CTA (a scratch buffer allocated and freed on `stream`) is summed in CTA order, so
 * the result is deterministic.  Cin 16, 32 or 64; Cout a multiple of 16 up to 64; Wout dividing
 * 64 and Hout Wout a multiple of 64: LSGD_EINVAL otherwise, LSGD_ENOMEM if the scratch cannot be
 * allocated, LSGD_EUNSUPPORTED without tcgen05. */
lsgd_status lsgd_conv_wgrad_bf16(const uint16_t* x, const uint16_t* dy, float* dW, int G, int B,
                                 int Hout, int Wout, int Cin, int Cout, int stride, void* stream);

/* A 3x3 convolution with zero padding 1 and stride s (1 or 2) for G independent groups on the
 * persistent implicit-GEMM tensor-core kernel, through the same code the ResNet-20 step runs
 * (Sec. A.2's network; 3x3 convolutions of He et al. 2016).  W [G][Cout][3][3][Cin] bf16.
 *  mode 0, forward:  out[g][b][oy][ox][co] = sum over kh, kw, ci of
 *          in[g][b][oy s + kh - 1][ox s + kw - 1][ci] W[g][co][kh][kw][ci]  (in zero outside the image)
 *          with in = x [G][B][Hin][Win][Cin] and out = y [G][B][Hout][Wout][Cout], Hout =
 *          (Hin - 1) / s + 1; Cin < 16 runs the stem form (image and weights padded with zero
 *          channels to 16).
 *  mode 1, data gradient: out[g][b][iy][ix][ci] = sum over (oy, ox, kh, kw) with
 *          iy = oy s + kh - 1, ix = ox s + kw - 1 and co of in[g][b][oy][ox][co] W[g][co][kh][kw][ci]
 *          with in = dy [G][B][Hout][Wout][Cout] and out = dx [G][B][Hin][Win][Cin]; stride 1 as
 *          a convolution with the flipped, transposed weights, stride 2 as four parity phases.
 * bf16 operands, fp32 accumulation; `out` fp32, fully overwritten.  Device pointers, in and W
 * 16-byte aligned, asynchronous on `stream`; scratch (the padded stem operands or the flipped
 * weights) is allocated and freed on `stream`.  LSGD_EINVAL on bad arguments, LSGD_EUNSUPPORTED
 * for shapes the kernel does not take (it needs 16, 32 or 64 channels per tap, Cout and Cin (mode
 * 1) of 16, 32 or 64, and an output whose whole rows tile into 128-pixel blocks), LSGD_ENOMEM if
 * the scratch cannot be allocated. */
lsgd_status lsgd_conv3x3_bf16(int mode, const uint16_t* in, const uint16_t* W, float* out, int G,
                              int B, int Hin, int Win, int Cin, int Cout, int stride,
                              void* stream);

/* The forward 3x3 convolution of lsgd_conv3x3_bf16 (mode 0) fused with the per-worker BatchNorm
 * statistics of its output (Sec. A.4; the first half of the conv -> BN -> ReLU unit of Sec. A.2's
 * ResNet-20), as the ResNet-20 training step computes them: y [G][B][Hout][Wout][Cout] fp32 as in
 * mode 0, and mean[G][Cout], rstd[G][Cout] = 1 / sqrt(biased variance + 1e-5) over the B Hout Wout
 * output positions of each group.  Each epilogue warp of the convolution keeps a running (count,
 * mean, sum of squared deviations) per channel, combining the two-pass moments of its 32 rows of
 * every 128-pixel tile in tile order by Chan et al.'s formula; a second kernel combines the
 * warps' partials in a fixed order, so the result is deterministic.  Same operands, alignment and shapes as mode 0 with
 * Cout <= 64; mean and rstd fp32 device arrays.  Scratch (the stem operands and the partials) is
 * allocated and freed on `stream`.  LSGD_EINVAL on bad arguments, LSGD_EUNSUPPORTED for shapes the
 * kernel does not take, LSGD_ENOMEM if the scratch cannot be allocated. */
lsgd_status lsgd_conv3x3_bn_bf16(const uint16_t* x, const uint16_t* W, float* y, float* mean,
                                 float* rstd, int G, int B, int Hin, int Win, int Cin, int Cout,
                                 int stride, void* stream);

/* lsgd_batchnorm_stats for callers that cannot allocate device memory during a run: a program
 * whose device memory is all handed to its own caching pool (an allocation would fail, or force
 * the pool to give memory back and stall), or a latency-critical loop that fixes its memory use at
 * start-up.  No counterpart in the paper: the method never allocates.  Same arguments and results
 * as lsgd_batchnorm_stats; the chunk partials go to a fixed 4 MiB array in the library's device
 * image (2^20 floats, kept on every GPU that loads the library until the process exits), so
 * G x ceil(P / 1024) x C x 2 must not exceed 1048576 (LSGD_EINVAL with a message otherwise).
 * No cudaMalloc / cudaFree / allocating call of any kind.  The first call on a device looks up
 * the array's device address with that device current (make that first call before any stream
 * capture).  All calls share the array: calls that may overlap on the GPU (other streams, other
 * host threads) race and must be ordered by the caller.  Nothing needs clearing between calls:
 * each call overwrites every partial it reads. */
lsgd_status lsgd_batchnorm_stats_noalloc(const float* y, int64_t P, int C, int G, float* mean,
                                         float* rstd, void* stream);

/* Worker mini-batch indices for one step into dst [K][B] int32 (device), as lsgd_local_step. */
lsgd_status lsgd_sample_indices(int32_t* dst, uint64_t seed, int64_t step, int K, int B, int64_t N,
                                void* stream);

#ifdef __cplusplus
}
#endif
#endif /* LSGD_H */
