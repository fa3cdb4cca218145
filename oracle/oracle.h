/* Oracle for the local / post-local SGD hot path -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, single-threaded restatement of "Don't Use Large Mini-Batches, Use Local SGD"
 * (Lin, Stich, Patel, Jaggi): mini-batch SGD (Eq. 1), local SGD (Eq. 2, Algorithm 1), post-local
 * SGD (the H_(t) switch of Sec. 3, Algorithm 2), local momentum (Sec. C.3.1, with the Nesterov /
 * no-dampening choice of Sec. A.4), weight decay (Sec. A.4), the large-batch learning-rate schemes
 * (Sec. A.3) and step decay (Sec. 4 / A.4).  Everything is computed in fp64; in "bf16" mode the
 * GEMM operands are rounded to bf16 exactly where the accelerated path stores them in bf16.
 *
 * Only tests/, the package smoke check and the benchmark's CPU-baseline leg may load this library.
 * It shares no code with the CUDA path and imports nothing from it.
 */
#ifndef LSGD_ORACLE_H
#define LSGD_ORACLE_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ORACLE_MAX_LAYERS 8

enum { ORACLE_DENSE = 0, ORACLE_LSQ = 1, ORACLE_RESNET20 = 2 };
enum { ORACLE_INIT_ZERO = 0, ORACLE_INIT_HE = 1 };

typedef struct {
  int kind;                             /* ORACLE_DENSE / ORACLE_LSQ / ORACLE_RESNET20 */
  int n_layers;                         /* dense layers (DENSE, LSQ) */
  int widths[ORACLE_MAX_LAYERS + 1];    /* widths[0] = input dim, widths[n_layers] = outputs */
  int has_bias;                         /* dense layers carry a bias vector */
  int bf16;                             /* 1: GEMM operands rounded to bf16 (RNE of the fp32 value) */
  int K, B, H;                          /* workers, local mini-batch, local steps per round */
  int64_t t_switch;                     /* post-local switch step t' (<0: local SGD from step 0) */
  int64_t T;                            /* total local steps of the run */
  int64_t N;                            /* dataset size */
  double base_lr;                       /* eta */
  int scale_by_K;                       /* eta_hat = K * eta */
  double warmup_epochs;                 /* linear warm-up length (0 = none) */
  int n_milestones;
  double milestones[4];                 /* fractions of T at which lr is multiplied by decay */
  double decay;
  double momentum;                      /* m (0 = plain SGD) */
  int nesterov;
  double weight_decay;
  uint64_t seed;
  /* ResNet-20 geometry (kind == ORACLE_RESNET20) */
  int in_h, in_w, in_c, n_classes, base_ch, res_blocks; /* res_blocks: basic blocks per stage */
  /* hierarchical local SGD (Sec. D): blocks of hier_block consecutive workers average after every
     H-step round, all K workers after every hier_rounds-th round (hier_block = 0: off) */
  int hier_block, hier_rounds;
  /* compressed averaging (Sec. B.3): 0 none, 1 signSGD variant (Algorithm 4: sign local steps,
     sign-compressed model differences), 2 EF-signSGD (Algorithm 5: error-feedback memory) */
  int compress;
  /* global momentum (Sec. C.3.1): > 0 applies momentum m_g to the averaged model difference */
  double global_momentum;
  /* local-step warm-up (Sec. C, "warm-up of the number of local SGD steps"; Sec. 4's ImageNet
     runs): the round that starts in epoch e < h_warmup_epochs has ORACLE_HWARM_* length instead
     of H */
  int h_warmup;
  double h_warmup_epochs;
  /* ORACLE_SAMPLE_SHARDS: static contiguous shards, uniform with replacement;
     ORACLE_SAMPLE_RESHUFFLE: a fresh global permutation every epoch, disjoint worker partitions,
     each worker passing through its partition in order (Sec. 4 / A.4 training procedure) */
  int sampling;
} oracle_cfg;

enum { ORACLE_HWARM_NONE = 0, ORACLE_HWARM_LINEAR = 1, ORACLE_HWARM_EXPONENTIAL = 2,
       ORACLE_HWARM_CONSTANT = 3 };
enum { ORACLE_SAMPLE_SHARDS = 0, ORACLE_SAMPLE_RESHUFFLE = 1 };

enum { ORACLE_COMPRESS_NONE = 0, ORACLE_COMPRESS_SIGN = 1, ORACLE_COMPRESS_EF_SIGN = 2 };

enum { ORACLE_SYNC_NONE = 0, ORACLE_SYNC_BLOCK = 1, ORACLE_SYNC_GLOBAL = 2 };

int64_t oracle_num_params(const oracle_cfg* c);
void oracle_weight_decay_mask(const oracle_cfg* c, uint8_t* mask);
void oracle_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]);
void oracle_sample_indices(const oracle_cfg* c, int k, int64_t s, int32_t* out);
/* Epoch of local step s: floor(s K B / N) (samples all workers accessed before it, over N). */
int64_t oracle_epoch(const oracle_cfg* c, int64_t s);
/* Length of the local-SGD round that starts at step s0. */
int64_t oracle_round_length(const oracle_cfg* c, int64_t s0);
/* pi_e(i): the epoch-e permutation of [0, N) of the reshuffling sampler. */
int64_t oracle_permute(const oracle_cfg* c, int64_t e, int64_t i);
void oracle_init_params(const oracle_cfg* c, int init_kind, double* w);
double oracle_loss_grad(const oracle_cfg* c, const double* w, const float* X, const int32_t* y,
                        const float* t, const int32_t* idx, int B, double* grad);
void oracle_sgd_update(const oracle_cfg* c, double lr, double* w, double* u, const double* g);
double oracle_lr(const oracle_cfg* c, int64_t s);
int oracle_is_round_end(const oracle_cfg* c, int64_t s);
int oracle_sync_kind(const oracle_cfg* c, int64_t s);
void oracle_average(int K, int64_t d, double* W);
void oracle_block_average(int K, int block, int64_t d, double* W);
void oracle_run(const oracle_cfg* c, const float* X, const int32_t* y, const float* t, double* W,
                double* U, int64_t s0, int64_t n_steps, double* losses, int64_t* n_syncs);
/* Local / post-local SGD with the synchronisation state of the compressed and global-momentum
 * variants: Wref [d] the synchronised model at the start of the round (NULL: taken from W[0]),
 * E [K][d] the error-feedback memories, Ug [d] the global momentum (NULL: zeros / not kept). */
void oracle_run_ext(const oracle_cfg* c, const float* X, const int32_t* y, const float* t,
                    double* W, double* U, double* Wref, double* E, double* Ug, int64_t s0,
                    int64_t n_steps, double* losses, int64_t* n_global, int64_t* n_block);
/* As oracle_run, also counting the block averages of hierarchical local SGD. */
void oracle_run_counted(const oracle_cfg* c, const float* X, const int32_t* y, const float* t,
                        double* W, double* U, int64_t s0, int64_t n_steps, double* losses,
                        int64_t* n_global, int64_t* n_block);
void oracle_run_minibatch(const oracle_cfg* c, const float* X, const int32_t* y, const float* t,
                          double* w, double* u, int64_t s0, int64_t n_steps, double* losses);
double oracle_eval_loss(const oracle_cfg* c, const double* w, const float* X, const int32_t* y,
                        const float* t, int64_t n);
double oracle_bf16_round(double x);

#ifdef __cplusplus
}
#endif
#endif
