// Runtime and C ABI of the local / post-local SGD hot path (declared in include/lsgd.h).
//
// K workers are simulated as K replicas in one replica-major arena: fp32 master weights W, local
// momentum U and gradients G, each [K][d_pad], plus a bf16 shadow Wb of W in BF16 mode (the GEMM
// operand).  Every per-replica tensor starts 256-byte aligned, so one rank-3 TMA map per operand
// (replica = outermost dimension) covers all K replicas.  A local step (Eq. 2 left, Algorithm 1's
// inner loop) is a fixed sequence of kernel launches on the context's stream with no host
// synchronisation; the K-way average (Eq. 2 right) is one kernel.
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <array>
#include <utility>
#include <algorithm>
#include <cstring>
#include <string>
#include <vector>

#include "../../include/lsgd.h"
#include "lsgd_internal.h"
#include "resnet.h"

namespace {

thread_local std::string g_last_error;

int64_t round_up(int64_t v, int64_t m) { return (v + m - 1) / m * m; }

struct Seg {
  int64_t canon, pad, len;
};

struct DenseLayer {
  int in, out, ld_in, ld_out;
  int64_t w_off, b_off;  // padded per-replica offsets (b_off < 0: no bias)
  bool tc;               // this layer's products run on tcgen05
  lsgd::TcOperand fwdA, fwdB, dgA, dgB, wgA, wgB;
};

}  // namespace

namespace lsgd {
void set_last_error(const std::string& msg) { g_last_error = msg; }
}  // namespace lsgd

// A round of the local-step warm-up schedule: its first step and length (len <= 0: unknown).
struct RoundCursor {
  int64_t start = 0;
  int64_t len = 0;
};

struct lsgd_ctx {
  lsgd_config cfg;
  lsgd_allocator alloc{};
  bool have_alloc = false;
  cudaStream_t stream = nullptr;
  int64_t d = 0, d_pad = 0, T = 0, shard = 0;
  int D = 0, C = 0;  // input width, outputs
  bool bf16 = false, lsq = false, resnet = false;
  bool fused = false;  // update applied in the weight-gradient epilogues (see lsgd_config)
  bool head = false;   // last layer + loss by the two classifier-head kernels (bf16, few classes)
  float* loss_slot_now = nullptr;  // this step's entry of the loss history (head path)
  std::vector<DenseLayer> layers;
  std::vector<Seg> segs;
  int64_t wd_period = 0, wd_end = 0;
  std::vector<void*> allocs;
  float *W = nullptr, *U = nullptr, *G = nullptr;
  uint16_t* Wb = nullptr;
  float* X = nullptr;
  int32_t* y = nullptr;
  float* t = nullptr;
  bool have_data = false;
  int32_t* idx = nullptr;
  int32_t* yb = nullptr;
  float* tb = nullptr;
  // host mini-batches (lsgd_local_step_batch): two staging buffers filled on a copy stream, so
  // the next batch's host-to-device copy overlaps the current step
  float* simt_ws = nullptr;  // split-K partials of the SIMT forward products (fp32 mode)
  int64_t simt_ws_floats = 0;
  float* xstage[2] = {nullptr, nullptr};
  void* lstage[2] = {nullptr, nullptr};  // labels (int32) or targets (fp32)
  cudaStream_t copy_stream = nullptr;
  cudaEvent_t stage_copied[2] = {nullptr, nullptr};  // the copy into the buffer has landed
  cudaEvent_t stage_free[2] = {nullptr, nullptr};    // the gather that read the buffer is done
  bool stage_used[2] = {false, false};
  int stage_next = 0;
  std::vector<void*> act;  // act[l]: input of dense layer l, [K][B][ld] operand dtype
  float* logits = nullptr;
  int ld_logits = 0;
  // split-K partial products of a narrow top layer's forward (logit_splits of them), or none
  float* logit_parts = nullptr;
  int logit_splits = 0;
  // output gradients: ping-pong buffers, and a third that keeps the top layer's while the layers
  // below use the first two (its update joins the last update launch)
  void* dz[3] = {nullptr, nullptr, nullptr};
  int ld_dz = 0;
  float* loss_hist = nullptr;
  int64_t loss_cap = 0;
  float* row_loss = nullptr;  // [K][B] scratch for evaluation
  int* flag = nullptr;
  int64_t step = 0, syncs = 0, block_syncs = 0, launches = 0;
  std::string err;
  lsgd::ResNetPlan* rn = nullptr;
  // tracing (lsgd_profile_*)
  // synchronisation state of the compressed / global-momentum averages
  float* wref = nullptr;   // [d_pad] model at the start of the round
  float* E = nullptr;      // [K][d_pad] error-feedback memories
  float* ug = nullptr;     // [d_pad] global momentum
  float* pnorm = nullptr;  // [K] ||Delta_k||_1 / d
  float* l1part = nullptr; // [K][l1_chunks] partial sums
  RoundCursor cursor;       // the round lsgd_run last stood in (local-step warm-up)
  // every replica holds the same parameters (after creation, a global average or a broadcast
  // lsgd_set_params); lets a step that ends with the average read each weight tile once
  bool synced = true;
  // the parameter segments a weight-gradient + update + average launch does not cover (the
  // biases and the classifier head's tensors), averaged by a small kernel after it
  lsgd::AvgSegments avg_segs{};
  // the weight matrices that launch does cover: after it only replica 0 holds them (and their
  // bf16 shadow) -- `lazy` -- until the next step rewrites every replica or materialize() copies
  // replica 0 to the others for a reader outside the step
  lsgd::AvgSegments wgrad_segs{};
  bool lazy = false;
  bool prof_on = false;
  std::vector<cudaEvent_t> prof_pool;
  size_t prof_used = 0;
  std::vector<std::array<int64_t, 3>> prof_spans;  // (phase, start event, end event)
};

namespace {

lsgd_status fail(lsgd_ctx* c, lsgd_status st, const std::string& msg) {
  if (c) c->err = msg;
  g_last_error = msg;
  return st;
}

lsgd_status fail_cuda(lsgd_ctx* c, cudaError_t e, const char* what) {
  return fail(c, LSGD_ECUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

#define LSGD_TRY_CUDA(ctx, expr)                                  \
  do {                                                            \
    cudaError_t e__ = (expr);                                     \
    if (e__ != cudaSuccess) return fail_cuda((ctx), e__, #expr); \
  } while (0)

#define LSGD_LAUNCH(ctx, expr)                                    \
  do {                                                            \
    cudaError_t e__ = (expr);                                     \
    (ctx)->launches++;                                            \
    if (e__ != cudaSuccess) return fail_cuda((ctx), e__, #expr); \
  } while (0)

void* dalloc(lsgd_ctx* c, size_t bytes) {
  if (bytes == 0) bytes = 256;
  bytes = (size_t)round_up((int64_t)bytes, 256);
  void* p = nullptr;
  if (c->have_alloc) {
    p = c->alloc.alloc(c->alloc.user, bytes, (void*)c->stream);
  } else {
    if (cudaMallocAsync(&p, bytes, c->stream) != cudaSuccess) {
      cudaGetLastError();
      p = nullptr;
    }
  }
  if (!p) return nullptr;
  if (cudaMemsetAsync(p, 0, bytes, c->stream) != cudaSuccess) {
    cudaGetLastError();
  }
  c->allocs.push_back(p);
  return p;
}

void free_all(lsgd_ctx* c) {
  for (void* p : c->allocs) {
    if (c->have_alloc)
      c->alloc.free(c->alloc.user, p, (void*)c->stream);
    else
      cudaFreeAsync(p, c->stream);
  }
  c->allocs.clear();
}

// ---- tracing: an event at each phase boundary, paired into spans ----
int64_t prof_mark(lsgd_ctx* c) {
  if (!c->prof_on) return -1;
  if (c->prof_used == c->prof_pool.size()) {
    cudaEvent_t e;
    if (cudaEventCreate(&e) != cudaSuccess) {
      cudaGetLastError();
      return -1;
    }
    c->prof_pool.push_back(e);
  }
  cudaEventRecord(c->prof_pool[c->prof_used], c->stream);
  return (int64_t)c->prof_used++;
}

void prof_span(lsgd_ctx* c, int phase, int64_t a, int64_t b) {
  if (c->prof_on && a >= 0 && b >= 0) c->prof_spans.push_back({phase, a, b});
}

// ---- schedules (Sec. A.3, A.4 and Sec. 3) ----
double lr_at(const lsgd_config& cfg, int64_t T, int64_t s) {
  const double eta = cfg.lr.base_lr;
  const double eta_hat = cfg.lr.scale_by_K ? eta * cfg.K : eta;
  double lr = eta_hat;
  if (cfg.lr.warmup_epochs > 0.0 && eta_hat != eta) {
    const double steps_per_epoch = (double)cfg.N / ((double)cfg.K * cfg.B_loc);
    const double inc = (eta_hat - eta) / (cfg.lr.warmup_epochs * steps_per_epoch);
    const double v = eta + (double)s * inc;
    lr = v < eta_hat ? v : eta_hat;
  }
  for (int i = 0; i < cfg.lr.n_milestones; ++i)
    if (s >= (int64_t)std::floor(cfg.lr.milestone_frac[i] * (double)T)) lr *= cfg.lr.decay;
  return lr;
}

// Epoch of step s: the samples all workers used before it, over N.
int64_t epoch_of(const lsgd_config& cfg, int64_t s) {
  return s * (int64_t)cfg.K * cfg.B_loc / cfg.N;
}

// Local-step warm-up (Sec. C; Sec. 4's ImageNet runs): the round that starts at step s0, in epoch
// e < P, has 1 + floor((H - 1) e / P) steps (linear), min(H, 2^floor(e log2 H / P)) (exponential)
// or 1 (constant); H from epoch P on.
int64_t round_length(const lsgd_config& cfg, int64_t s0) {
  if (cfg.h_warmup == LSGD_HWARM_NONE) return cfg.H;
  const double e = (double)epoch_of(cfg, s0), P = cfg.h_warmup_epochs;
  if (e >= P) return cfg.H;
  if (cfg.h_warmup == LSGD_HWARM_LINEAR) return 1 + (int64_t)std::floor((double)(cfg.H - 1) * e / P);
  if (cfg.h_warmup == LSGD_HWARM_EXPONENTIAL) {
    const double len = std::pow(2.0, std::floor(e * std::log2((double)cfg.H) / P));
    return len < (double)cfg.H ? (int64_t)len : cfg.H;
  }
  return 1;
}

// Whether step s ends a round: every step before the switch t' (post-local SGD, Sec. 3), then
// rounds of H steps (of round_length steps with a local-step warm-up, walked forward from the
// round `cur` last stood in); the last step of the run always does.
bool round_end(const lsgd_config& cfg, int64_t T, int64_t s, RoundCursor* cur) {
  if (s == T - 1) return true;
  if (cfg.t_switch >= 0 && s < cfg.t_switch) return true;
  const int64_t start = cfg.t_switch > 0 ? cfg.t_switch : 0;
  if (cfg.h_warmup == LSGD_HWARM_NONE) return ((s + 1 - start) % cfg.H) == 0;
  if (cur->len <= 0 || cur->start > s) *cur = RoundCursor{start, round_length(cfg, start)};
  while (s >= cur->start + cur->len) {
    cur->start += cur->len;
    cur->len = round_length(cfg, cur->start);
  }
  return s == cur->start + cur->len - 1;
}

// Average ending step s: 0 none, 1 block (hierarchical), 2 global (Sec. 3 and Sec. D).
int sync_kind_at(const lsgd_config& cfg, int64_t T, int64_t s, RoundCursor* cur) {
  if (!round_end(cfg, T, s, cur)) return 0;
  if (cfg.hier_block <= 0 || s == T - 1) return 2;
  if (cfg.t_switch >= 0 && s < cfg.t_switch) return 2;
  const int64_t start = cfg.t_switch > 0 ? cfg.t_switch : 0;
  const int64_t r = (s + 1 - start) / cfg.H;
  return (r % std::max(1, cfg.hier_rounds) == 0) ? 2 : 1;
}

bool force_simt() {
  const char* e = std::getenv("LSGD_FORCE_SIMT");
  return e && e[0] == '1';
}

// ---- dense model ----
lsgd_status build_dense_layout(lsgd_ctx* c) {
  const lsgd_model& m = c->cfg.model;
  int64_t off = 0, canon = 0;
  for (int l = 0; l < m.n_layers; ++l) {
    DenseLayer L{};
    L.in = m.widths[l];
    L.out = m.widths[l + 1];
    L.ld_in = (int)round_up(L.in, 8);
    L.ld_out = (int)round_up(L.out, 8);
    L.w_off = off;
    c->segs.push_back({canon, off, (int64_t)L.in * L.out});
    canon += (int64_t)L.in * L.out;
    off = round_up(off + (int64_t)L.in * L.out, 64);
    if (!c->lsq) {
      L.b_off = off;
      c->segs.push_back({canon, off, L.out});
      canon += L.out;
      off = round_up(off + L.out, 64);
    } else {
      L.b_off = -1;
    }
    c->layers.push_back(L);
  }
  c->d = canon;
  c->d_pad = round_up(off, 64);
  c->wd_period = 0;
  c->wd_end = c->d_pad;
  return LSGD_OK;
}

lsgd_status make_tc_maps(lsgd_ctx* c) {
  const int K = c->cfg.K, B = c->cfg.B_loc;
  for (size_t l = 0; l < c->layers.size(); ++l) {
    DenseLayer& L = c->layers[l];
    L.tc = false;
    if (!c->bf16 || force_simt() || !lsgd::tc_available()) continue;
    const uint16_t* Wb_l = c->Wb + L.w_off;
    const void* a_in = c->act[l];
    bool ok = true;
    // forward: A = act [K][B][ld_in] (K-major), B = W [K][out][in] (K-major)
    const int bn = lsgd::tc_tile_n(L.in);
    ok &= lsgd::make_tma_map_bf16(&L.fwdA.map, a_in, L.in, B, K, L.ld_in, (uint64_t)B * L.ld_in, 64,
                                  lsgd::kTcTileM);
    ok &= lsgd::make_tma_map_bf16(&L.fwdB.map, Wb_l, L.in, L.out, K, L.in, c->d_pad, 64, bn);
    L.fwdA.mn_major = false;
    L.fwdA.box_rows = lsgd::kTcTileM;
    L.fwdB.mn_major = false;
    L.fwdB.box_rows = bn;
    // weight gradient: A = dZ as [K][B][out] read MN-major (M = out), B = act read MN-major (N = in)
    // The dz buffer used for layer l alternates; both dz buffers share one layout, so the maps are
    // rebuilt per call from the right base (cheap host work, see run_dense_backward).
    (void)a_in;
    L.tc = ok;
  }
  return LSGD_OK;
}

// The top layer's fused update joins the last update launch (that of layers 1 and 0) rather than
// running alone: with three or more layers updated by the weight-gradient kernel and no classifier
// head.  Its output gradient then stays in dz[2] while the layers below use dz[0] and dz[1], and
// nothing between its own backward and that launch reads its weights (the layers below read only
// theirs), so the result is the same.
bool defer_top_update(const lsgd_ctx* c) {
  return c->fused && !c->head && c->layers.size() >= 3;
}

lsgd_status alloc_dense(lsgd_ctx* c) {
  const int K = c->cfg.K, B = c->cfg.B_loc;
  const size_t esz = c->bf16 ? 2 : 4;
  const int L = (int)c->layers.size();
  c->act.resize(L);
  int max_ld = 8;
  for (int l = 0; l < L; ++l) {
    c->act[l] = dalloc(c, (size_t)K * B * c->layers[l].ld_in * esz);
    if (!c->act[l]) return fail(c, LSGD_ENOMEM, "activation buffer allocation failed");
    max_ld = std::max(max_ld, c->layers[l].ld_out);
  }
  c->ld_logits = c->layers[L - 1].ld_out;
  c->logits = (float*)dalloc(c, (size_t)K * B * c->ld_logits * 4);
  c->ld_dz = max_ld;
  for (int i = 0; i < 2; ++i) c->dz[i] = dalloc(c, (size_t)K * B * max_ld * esz);
  if (!c->logits || !c->dz[0] || !c->dz[1]) return fail(c, LSGD_ENOMEM, "gradient buffer allocation failed");
  return LSGD_OK;
}

lsgd_status init_dense_params(lsgd_ctx* c) {
  if (c->cfg.model.init == LSGD_INIT_HE) {
    for (size_t l = 0; l < c->layers.size(); ++l) {
      const DenseLayer& L = c->layers[l];
      LSGD_LAUNCH(c, lsgd::launch_init_normal(c->W + L.w_off, (int64_t)L.in * L.out,
                                              std::sqrt(2.0 / L.in), c->cfg.seed, (uint32_t)l,
                                              c->stream));
    }
  }
  return LSGD_OK;
}

// GEMM helpers: choose the tcgen05 kernel for bf16 layers that have maps, else SIMT.
lsgd_status gemm(lsgd_ctx* c, const lsgd::GemmArgs& g) {
  LSGD_LAUNCH(c, lsgd::launch_gemm_simt(g, c->stream));
  return LSGD_OK;
}

lsgd_status tc_gemm(lsgd_ctx* c, const lsgd::TcGemmArgs& g) {
  LSGD_LAUNCH(c, lsgd::launch_gemm_tc(g, c->stream));
  return LSGD_OK;
}

// Forward of every dense layer for `groups` groups.  Weights come from replica (w_g0 + g * w_gmul).
lsgd_status dense_forward(lsgd_ctx* c, int groups, int w_g0, int w_gmul, bool skip_last = false) {
  const int B = c->cfg.B_loc;
  const int L = (int)c->layers.size();
  const void* Wop = c->bf16 ? (const void*)c->Wb : (const void*)c->W;
  const size_t esz = c->bf16 ? 2 : 4;
  for (int l = 0; l < (skip_last ? L - 1 : L); ++l) {
    const DenseLayer& Ly = c->layers[l];
    const bool last = l == L - 1;
    void* out = last ? (void*)c->logits : c->act[l + 1];
    const int ld_out = last ? c->ld_logits : c->layers[l + 1].ld_in;
    const bool out_bf16 = last ? false : c->bf16;
    const int epi = c->lsq ? lsgd::EPI_STORE : (last ? lsgd::EPI_BIAS : lsgd::EPI_BIAS_RELU);
    if (Ly.tc && w_gmul == 1 && w_g0 == 0) {
      lsgd::TcGemmArgs t{};
      t.M = B;
      t.N = Ly.out;
      t.Kd = Ly.in;
      t.G = groups;
      t.A = Ly.fwdA;
      t.B = Ly.fwdB;
      t.C = out;
      t.c_rs = ld_out;
      t.c_gs = (int64_t)B * ld_out;
      t.c_bf16 = out_bf16;
      t.epi = epi;
      t.bias = Ly.b_off >= 0 ? c->W + Ly.b_off : nullptr;
      t.bias_gs = c->d_pad;
      // every replica holds the same weights: all read replica 0's, which stay in L2
      t.b_shared = (c->synced && groups == c->cfg.K && c->cfg.K > 1) ? 1 : 0;
      if (last && c->logit_splits > 1 && epi == lsgd::EPI_BIAS) {
        // split-K partial products, then their sum in split order plus the bias
        const int64_t sstride = (int64_t)c->cfg.K * B * ld_out;
        t.splits = c->logit_splits;
        t.c_split_stride = sstride;
        t.C = c->logit_parts;
        t.epi = lsgd::EPI_STORE;
        t.bias = nullptr;
        lsgd_status st = tc_gemm(c, t);
        if (st != LSGD_OK) return st;
        LSGD_LAUNCH(c, lsgd::launch_split_bias_sum(c->logit_parts, c->logit_splits, sstride,
                                                   Ly.b_off >= 0 ? c->W + Ly.b_off : nullptr,
                                                   c->d_pad, groups, B, Ly.out, ld_out,
                                                   (float*)out, c->stream));
        continue;
      }
      lsgd_status st = tc_gemm(c, t);
      if (st != LSGD_OK) return st;
      continue;
    }
    lsgd::GemmArgs g{};
    g.M = B;
    g.N = Ly.out;
    g.Kd = Ly.in;
    g.G = groups;
    g.A = c->act[l];
    g.a_rs = Ly.ld_in;
    g.a_cs = 1;
    g.a_gs = (int64_t)B * Ly.ld_in;
    g.a_bf16 = c->bf16;
    g.B = (const char*)Wop + ((int64_t)w_g0 * c->d_pad + Ly.w_off) * esz;
    g.b_rs = 1;
    g.b_cs = Ly.in;
    g.b_gs = (int64_t)w_gmul * c->d_pad;
    g.b_bf16 = c->bf16;
    g.C = out;
    g.c_rs = ld_out;
    g.c_gs = (int64_t)B * ld_out;
    g.c_bf16 = out_bf16;
    g.epi = epi;
    g.bias = Ly.b_off >= 0 ? c->W + (int64_t)w_g0 * c->d_pad + Ly.b_off : nullptr;
    g.bias_gs = (int64_t)w_gmul * c->d_pad;
    g.ws = c->simt_ws;
    g.ws_floats = c->simt_ws_floats;
    lsgd_status st = gemm(c, g);
    if (st != LSGD_OK) return st;
  }
  (void)esz;
  return LSGD_OK;
}

// The classifier-head kernels' view of the last layer (forward + loss and backward share it).
lsgd::HeadArgs head_args(lsgd_ctx* c) {
  const DenseLayer& Ly = c->layers.back();
  lsgd::HeadArgs h{};
  h.C = Ly.out;
  h.B = c->cfg.B_loc;
  h.in = Ly.in;
  h.reps = c->cfg.K;
  h.rep_stride = c->d_pad;
  h.w_off = Ly.w_off;
  h.b_off = Ly.b_off;
  h.act = (const uint16_t*)c->act[c->layers.size() - 1];
  h.ld_in = Ly.ld_in;
  h.Wb = c->Wb;
  h.W = c->W;
  h.labels = c->yb;
  h.dz = (uint16_t*)c->dz[0];
  h.ld_dz = c->ld_dz;
  h.row_loss = c->row_loss;
  h.b_prev_off = -1;
  return h;
}

// Backward of every dense layer, last to first: data gradient (it reads this layer's weights, so
// it runs before a fused update may change them), weight gradient, bias gradient.
lsgd_status dense_backward(lsgd_ctx* c, bool avg) {
  const int K = c->cfg.K, B = c->cfg.B_loc;
  const int L = (int)c->layers.size();
  const void* Wop = c->bf16 ? (const void*)c->Wb : (const void*)c->W;
  const size_t esz = c->bf16 ? 2 : 4;
  lsgd::SgdParams sgd{};
  if (c->fused) {
    sgd.lr = (float)lr_at(c->cfg, c->T, c->step);
    sgd.mom = (float)c->cfg.momentum;
    sgd.wd = (float)c->cfg.weight_decay;
    sgd.nesterov = c->cfg.nesterov;
    sgd.sign = c->cfg.compress == LSGD_COMPRESS_SIGN;
  }
  auto sgd_at = [&](int64_t off) {
    lsgd::SgdParams p = sgd;
    p.w = c->W + off;
    p.u = c->U ? c->U + off : nullptr;
    p.wb = c->Wb ? c->Wb + off : nullptr;
    return p;
  };
  // Tracing: with the fused update the weight-gradient launches are the update phase, the rest
  // is the backward phase; otherwise the caller times the whole backward as one span.
  int64_t e_prev = c->fused ? prof_mark(c) : -1;
  auto span = [&](int phase) {
    if (!c->fused) return;
    const int64_t e = prof_mark(c);
    prof_span(c, phase, e_prev, e);
    e_prev = e;
  };
  int cur = 0;
  int l_top = L - 1;
  int bias_done = -1;  // layer whose bias the last data-gradient GEMM already handled
  lsgd::WgradUpdateArgs wa{};  // fused weight-gradient + update layers not yet launched
  // the top layer's update waits for the last update launch (defer_top_update); its output
  // gradient stays in dz[0] and the layers below alternate between dz[1] and dz[2]
  const bool defer_top = defer_top_update(c) && c->dz[2] != nullptr;
  lsgd::WgradUpdateLayer top_layer{};
  bool top_pending = false;
  auto next_dz = [&](int b) { return defer_top ? (b == 1 ? 2 : 1) : 1 - b; };
  if (c->head) {
    // the last layer's weight / bias gradients and their update (its data gradient for the layer
    // below came with the head's forward kernel)
    lsgd::HeadArgs h = head_args(c);
    h.loss_mean = c->loss_slot_now;
    if (L > 1) {
      h.dz_prev = (uint16_t*)c->dz[1];
      h.ld_dz_prev = c->ld_dz;
      h.b_prev_off = c->layers[L - 2].b_off;  // the layer below's bias, from the stored dA
    }
    h.fused = c->fused ? 1 : 0;
    h.sgd = sgd;
    h.sgd.w = c->W;
    h.sgd.u = c->U;
    h.sgd.wb = c->Wb;
    h.grad = c->G;
    LSGD_LAUNCH(c, lsgd::launch_head_backward(h, c->stream));
    span(LSGD_PH_UPDATE);
    l_top = L - 2;
    cur = 1;
  }
  for (int l = l_top; l >= 0; --l) {
    const DenseLayer& Ly = c->layers[l];
    const void* dz = c->dz[cur];
    // read before this layer's data gradient sets bias_done for the layer below
    const bool bias_by_dgrad_above = bias_done == l;
    if (l > 0) {
      // data gradient dz_prev[j][i] = (sum_o dz[j][o] W[o][i]) * (act[j][i] > 0)
      void* dzp = c->dz[next_dz(cur)];
      if (Ly.tc) {
        lsgd::TcGemmArgs t{};
        t.M = B;
        t.N = Ly.in;
        t.Kd = Ly.out;
        t.G = K;
        bool ok = lsgd::make_tma_map_bf16(&t.A.map, dz, Ly.out, B, K, c->ld_dz, (uint64_t)B * c->ld_dz,
                                          64, lsgd::kTcTileM);
        ok &= lsgd::make_tma_map_bf16(&t.B.map, c->Wb + Ly.w_off, Ly.in, Ly.out, K, Ly.in, c->d_pad, 64, 64);
        if (!ok) return fail(c, LSGD_ECUDA, "TMA map encoding failed (dgrad)");
        t.A.mn_major = false;
        t.A.box_rows = lsgd::kTcTileM;
        t.B.mn_major = true;
        t.B.box_rows = 64;
        t.b_shared = (c->synced && K > 1) ? 1 : 0;  // identical replicas: one weight copy
        t.C = dzp;
        t.c_rs = c->ld_dz;
        t.c_gs = (int64_t)B * c->ld_dz;
        t.c_bf16 = c->bf16;
        t.epi = lsgd::EPI_MASK;
        t.mask = c->act[l];
        t.mask_rs = Ly.ld_in;
        t.mask_gs = (int64_t)B * Ly.ld_in;
        t.mask_bf16 = c->bf16;
        const DenseLayer& below = c->layers[l - 1];
        if (below.b_off >= 0 && B <= lsgd::kTcTileM) {
          // the whole mini-batch is one tile: the epilogue also sums the stored result over rows,
          // which is the bias gradient of the layer below, and updates that bias
          t.bias_colsum = true;
          t.bias_gs = c->d_pad;
          if (c->fused)
            t.bsgd = sgd_at(below.b_off);
          else
            t.bias_grad = c->G + below.b_off;
          bias_done = l - 1;
        }
        lsgd_status st = tc_gemm(c, t);
        if (st != LSGD_OK) return st;
      } else {
        lsgd::GemmArgs g{};
        g.M = B;
        g.N = Ly.in;
        g.Kd = Ly.out;
        g.G = K;
        g.A = dz;
        g.a_rs = c->ld_dz;
        g.a_cs = 1;
        g.a_gs = (int64_t)B * c->ld_dz;
        g.a_bf16 = c->bf16;
        g.B = (const char*)Wop + Ly.w_off * esz;
        g.b_rs = Ly.in;
        g.b_cs = 1;
        g.b_gs = c->d_pad;
        g.b_bf16 = c->bf16;
        g.C = dzp;
        g.c_rs = c->ld_dz;
        g.c_gs = (int64_t)B * c->ld_dz;
        g.c_bf16 = c->bf16;
        g.epi = lsgd::EPI_MASK;
        g.mask = c->act[l];
        g.mask_rs = Ly.ld_in;
        g.mask_gs = (int64_t)B * Ly.ld_in;
        g.mask_bf16 = c->bf16;
        lsgd_status st = gemm(c, g);
        if (st != LSGD_OK) return st;
      }
      span(LSGD_PH_BACKWARD);
    }
    // weight gradient G_W[o][i] = sum_j dz[j][o] act[j][i] (or, fused, the update it drives)
    if (Ly.tc) {
      lsgd::TcGemmArgs t{};
      t.M = Ly.out;
      t.N = Ly.in;
      t.Kd = B;
      t.G = K;
      bool ok = lsgd::make_tma_map_bf16(&t.A.map, dz, Ly.out, B, K, c->ld_dz, (uint64_t)B * c->ld_dz, 64, 64);
      ok &= lsgd::make_tma_map_bf16(&t.B.map, c->act[l], Ly.in, B, K, Ly.ld_in, (uint64_t)B * Ly.ld_in, 64, 64);
      if (!ok) return fail(c, LSGD_ECUDA, "TMA map encoding failed (wgrad)");
      t.A.mn_major = true;
      t.B.mn_major = true;
      t.A.box_rows = 64;
      t.B.box_rows = 64;
      t.c_rs = Ly.in;
      t.c_gs = c->d_pad;
      t.c_bf16 = false;
      if (c->fused) {
        // persistent weight-gradient + update kernel: parameters, momentum and the bf16 shadow
        // stream through shared memory by TMA in 128 x 32 chunks
        lsgd::WgradUpdateLayer& wl = wa.L[wa.nl];
        wl.M = Ly.out;
        wl.N = Ly.in;
        wl.A = t.A;
        wl.B = t.B;
        const lsgd::SgdParams sp = sgd_at(Ly.w_off);
        bool mok = lsgd::make_tma_map(&wl.wmap, sp.w, false, Ly.in, Ly.out, K, Ly.in, c->d_pad,
                                      32, 128, 128);
        if (sp.u)
          mok &= lsgd::make_tma_map(&wl.umap, sp.u, false, Ly.in, Ly.out, K, Ly.in, c->d_pad,
                                    32, 128, 128);
        if (sp.wb)
          mok &= lsgd::make_tma_map(&wl.wbmap, sp.wb, true, Ly.in, Ly.out, K, Ly.in, c->d_pad,
                                    32, 128, 64);
        if (!mok) return fail(c, LSGD_ECUDA, "TMA map encoding failed (fused update)");
        if (wa.nl == 0) wa.sgd = sp;
        ++wa.nl;
        if (defer_top && l == L - 1) {
          top_layer = wa.L[0];
          top_pending = true;
          wa.nl = 0;
        } else if (!(l == 1 && c->layers[0].tc)) {
          // Layer 1's update waits for layer 0's, so both go in one launch: nothing in between
          // writes the gradients they read (layer 0 has no data gradient) or reads the parameters
          // they change; a deferred top layer joins them last.
          if (top_pending && l == 0) {
            wa.L[wa.nl++] = top_layer;
            top_pending = false;
          }
          wa.Kd = B;
          wa.G = K;
          wa.avg = avg ? 1 : 0;
          wa.w_rep0 = (c->synced && K > 1) ? 1 : 0;  // one copy serves every replica
          LSGD_LAUNCH(c, lsgd::launch_wgrad_update(wa, c->stream));
          wa.nl = 0;
          span(LSGD_PH_UPDATE);
        }
      } else {
        t.C = c->G + Ly.w_off;
        t.epi = lsgd::EPI_STORE;
        lsgd_status st = tc_gemm(c, t);
        if (st != LSGD_OK) return st;
        span(LSGD_PH_UPDATE);
      }
    } else {
      lsgd::GemmArgs g{};
      g.M = Ly.out;
      g.N = Ly.in;
      g.Kd = B;
      g.G = K;
      g.A = dz;
      g.a_rs = 1;
      g.a_cs = c->ld_dz;
      g.a_gs = (int64_t)B * c->ld_dz;
      g.a_bf16 = c->bf16;
      g.B = c->act[l];
      g.b_rs = Ly.ld_in;
      g.b_cs = 1;
      g.b_gs = (int64_t)B * Ly.ld_in;
      g.b_bf16 = c->bf16;
      g.C = c->G + Ly.w_off;
      g.c_rs = Ly.in;
      g.c_gs = c->d_pad;
      g.c_bf16 = false;
      g.epi = lsgd::EPI_STORE;
      lsgd_status st = gemm(c, g);
      if (st != LSGD_OK) return st;
      span(LSGD_PH_UPDATE);
    }
    // the bias sums: unless the head's kernel (layer L - 2) or the data-gradient GEMM above did them
    if (Ly.b_off >= 0 && !(c->head && l == L - 2) && !bias_by_dgrad_above) {
      if (c->fused)
        LSGD_LAUNCH(c, lsgd::launch_colsum_update(dz, c->bf16, c->ld_dz, K, B, Ly.out, c->d_pad,
                                                  sgd_at(Ly.b_off), c->stream));
      else
        LSGD_LAUNCH(c, lsgd::launch_colsum(dz, c->bf16, c->ld_dz, K, B, Ly.out, c->G + Ly.b_off,
                                           c->d_pad, c->stream));
      span(LSGD_PH_BACKWARD);
    }
    if (l > 0) cur = next_dz(cur);
  }
  if (top_pending) return fail(c, LSGD_ESTATE, "deferred top-layer update was not launched");
  return LSGD_OK;
}

// Loss of the last layer's output for `groups` groups; dz into dz[0] unless eval.
lsgd_status dense_loss(lsgd_ctx* c, int groups, bool eval, float* loss_mean) {
  const int B = c->cfg.B_loc;
  void* dz = eval ? nullptr : c->dz[0];
  if (c->lsq) {
    LSGD_LAUNCH(c, lsgd::launch_lsq_loss(c->logits, c->ld_logits, c->tb, groups, B, dz, c->bf16,
                                         c->ld_dz, loss_mean, nullptr, c->row_loss, c->stream));
  } else {
    LSGD_LAUNCH(c, lsgd::launch_softmax_xent(c->logits, c->ld_logits, c->C, c->yb, groups, B, dz,
                                             c->bf16, c->ld_dz, loss_mean, nullptr, c->row_loss,
                                             c->stream));
  }
  return LSGD_OK;
}

lsgd_status do_update(lsgd_ctx* c) {
  const float lr = (float)lr_at(c->cfg, c->T, c->step);
  LSGD_LAUNCH(c, lsgd::launch_sgd_update(c->W, c->U, c->G, c->Wb, (int64_t)c->cfg.K * c->d_pad, lr,
                                         (float)c->cfg.momentum, c->cfg.nesterov,
                                         (float)c->cfg.weight_decay, c->wd_period, c->wd_end,
                                         c->stream, c->cfg.compress == LSGD_COMPRESS_SIGN));
  return LSGD_OK;
}

// Whether a step that ends with the global average can run it inside its update launches:
// dense bf16 model with the fused update on the tensor cores, plain averaging.
bool can_fuse_average(const lsgd_ctx* c) {
  return c->fused && !c->resnet && c->cfg.compress == LSGD_COMPRESS_NONE &&
         c->cfg.global_momentum <= 0.0;
}

// The step body after the inputs of this step are gathered into act[0] / yb / tb.  avg: the step
// ends with the K-way average, done by the update launches and the segment average
// (can_fuse_average must hold).
lsgd_status step_body(lsgd_ctx* c, int64_t e_start, bool avg = false) {
  const int K = c->cfg.K;
  float* loss_slot = c->loss_hist + (c->step % c->loss_cap) * K;
  lsgd_status st;
  const int64_t e_in = prof_mark(c);
  prof_span(c, LSGD_PH_INPUT, e_start, e_in);
  int64_t e_bwd;
  if (c->resnet) {
    st = lsgd::resnet_forward_backward(c->rn, c->W, c->Wb, c->G, c->d_pad, c->yb, loss_slot,
                                       c->stream, &c->launches);
    if (st != LSGD_OK) return fail(c, st, lsgd::resnet_last_error(c->rn));
    e_bwd = prof_mark(c);
    prof_span(c, LSGD_PH_FORWARD, e_in, e_bwd);
  } else {
    st = dense_forward(c, K, 0, 1, c->head);
    if (st != LSGD_OK) return st;
    const int64_t e_fwd = prof_mark(c);
    prof_span(c, LSGD_PH_FORWARD, e_in, e_fwd);
    if (c->head) {
      // the last layer's product, the loss, the logits gradient and the data gradient for the
      // layer below in one kernel; the mean loss is finished by the head's backward kernel
      lsgd::HeadArgs h = head_args(c);
      h.dz_prev = c->layers.size() > 1 ? (uint16_t*)c->dz[1] : nullptr;
      h.ld_dz_prev = c->ld_dz;
      LSGD_LAUNCH(c, lsgd::launch_head_forward(h, c->stream));
      c->loss_slot_now = loss_slot;
    } else {
      st = dense_loss(c, K, false, loss_slot);
    }
    if (st != LSGD_OK) return st;
    const int64_t e_loss = prof_mark(c);
    prof_span(c, LSGD_PH_LOSS, e_fwd, e_loss);
    st = dense_backward(c, avg);
    if (st != LSGD_OK) return st;
    e_bwd = prof_mark(c);
    if (!c->fused) prof_span(c, LSGD_PH_BACKWARD, e_loss, e_bwd);
  }
  if (!c->fused) {
    st = do_update(c);
    if (st != LSGD_OK) return st;
    prof_span(c, LSGD_PH_UPDATE, e_bwd, prof_mark(c));
  }
  c->step++;
  if (avg) {
    // the tensors the update launches did not average (biases, classifier head)
    LSGD_LAUNCH(c, lsgd::launch_average_segments(c->W, c->Wb, K, c->d_pad, c->avg_segs, c->stream));
    prof_span(c, LSGD_PH_AVERAGE, e_bwd, prof_mark(c));
    c->syncs++;
  }
  c->synced = avg || c->cfg.K == 1;
  // after the average only replica 0 holds the weight matrices; a plain step rewrites them all
  c->lazy = avg && c->cfg.K > 1;
  return LSGD_OK;
}

// Write replica 0's weight matrices (and bf16 shadow) to the other replicas if an average left
// them there alone: before anything outside the training step reads or changes single replicas.
lsgd_status materialize(lsgd_ctx* c) {
  if (!c->lazy) return LSGD_OK;
  LSGD_LAUNCH(c, lsgd::launch_broadcast_segments(c->W, c->Wb, c->cfg.K, c->d_pad, c->wgrad_segs,
                                                 c->stream));
  c->lazy = false;
  return LSGD_OK;
}

// Every check lsgd_create makes on a configuration before touching the GPU.
lsgd_status validate_config(const lsgd_config& c0) {
  if (c0.K < 1 || c0.B_loc < 1 || c0.H < 1) return fail(nullptr, LSGD_EINVAL, "K, B_loc and H must be >= 1");
  if (c0.N < c0.K) return fail(nullptr, LSGD_EINVAL, "N must be >= K");
  if (c0.K > 65535) return fail(nullptr, LSGD_EINVAL, "K must be <= 65535");
  if (c0.precision != LSGD_FP32 && c0.precision != LSGD_BF16)
    return fail(nullptr, LSGD_EINVAL, "precision must be LSGD_FP32 or LSGD_BF16");
  if (c0.N / c0.K * (int64_t)c0.K > 0x7fffffffLL) return fail(nullptr, LSGD_EINVAL, "N too large");
  if (c0.B_loc > 8192) return fail(nullptr, LSGD_EUNSUPPORTED, "B_loc must be <= 8192");
  if (c0.hier_block < 0 || (c0.hier_block > 0 && (c0.K % c0.hier_block || c0.hier_rounds < 1)))
    return fail(nullptr, LSGD_EINVAL, "hier_block must divide K and hier_rounds must be >= 1");
  if (c0.compress < LSGD_COMPRESS_NONE || c0.compress > LSGD_COMPRESS_EF_SIGN || c0.global_momentum < 0.0 ||
      ((c0.compress != LSGD_COMPRESS_NONE || c0.global_momentum > 0.0) && c0.hier_block > 0) ||
      (c0.compress != LSGD_COMPRESS_NONE && c0.global_momentum > 0.0))
    return fail(nullptr, LSGD_EINVAL,
                "compress and global_momentum exclude each other and hierarchical averaging");
  if (c0.compress != LSGD_COMPRESS_NONE && c0.K > 1024)
    return fail(nullptr, LSGD_EINVAL, "compress supports K <= 1024");
  if (c0.h_warmup < LSGD_HWARM_NONE || c0.h_warmup > LSGD_HWARM_CONSTANT ||
      c0.h_warmup_epochs < 0.0 || c0.sampling < LSGD_SAMPLE_SHARDS ||
      c0.sampling > LSGD_SAMPLE_RESHUFFLE)
    return fail(nullptr, LSGD_EINVAL, "bad h_warmup / h_warmup_epochs / sampling");
  if (c0.h_warmup != LSGD_HWARM_NONE && (c0.t_switch >= 0 || c0.hier_block > 0))
    return fail(nullptr, LSGD_EINVAL,
                "local-step warm-up replaces the post-local switch; not with hier_block");
  const lsgd_model& m = c0.model;
  if (m.kind == LSGD_MLP || m.kind == LSGD_LSQ) {
    if (m.n_layers < 1 || m.n_layers > LSGD_MAX_LAYERS)
      return fail(nullptr, LSGD_EINVAL, "n_layers must be in [1, LSGD_MAX_LAYERS]");
    for (int l = 0; l <= m.n_layers; ++l)
      if (m.widths[l] < 1) return fail(nullptr, LSGD_EINVAL, "layer widths must be >= 1");
    if (m.kind == LSGD_LSQ && (m.n_layers != 1 || m.widths[1] != 1))
      return fail(nullptr, LSGD_EINVAL, "least squares is one layer with one output");
    if (c0.precision == LSGD_BF16)
      for (int l = 0; l < m.n_layers; ++l)
        if (m.widths[l] % 8)
          return fail(nullptr, LSGD_EUNSUPPORTED, "BF16 dense layers need input widths divisible by 8");
  } else if (m.kind == LSGD_RESNET20) {
    std::string why;
    if (!lsgd::resnet_supported(c0, &why)) return fail(nullptr, LSGD_EUNSUPPORTED, why);
  } else {
    return fail(nullptr, LSGD_EINVAL, "unknown model kind");
  }

  return LSGD_OK;
}

// T: total_steps, else ceil(epochs N / (K B_loc)), at least 1.
int64_t total_steps_of(const lsgd_config& c0) {
  const int64_t T = c0.total_steps > 0
                        ? c0.total_steps
                        : (int64_t)std::ceil(c0.epochs * (double)c0.N / ((double)c0.K * c0.B_loc) - 1e-9);
  return T < 1 ? 1 : T;
}

void* input_buffer(lsgd_ctx* c) { return c->resnet ? lsgd::resnet_input(c->rn) : c->act[0]; }
int input_ld(lsgd_ctx* c) { return c->resnet ? c->D : c->layers[0].ld_in; }

}  // namespace

// =============================================================================================
extern "C" {

lsgd_status lsgd_create(const lsgd_config* cfg, const lsgd_allocator* alloc, void* cuda_stream,
                        lsgd_ctx** out) {
  if (!cfg || !out) return fail(nullptr, LSGD_EINVAL, "cfg and out must be non-NULL");
  const lsgd_config& c0 = *cfg;
  const lsgd_status vst = validate_config(c0);
  if (vst != LSGD_OK) return vst;
  const lsgd_model& m = c0.model;
  lsgd_ctx* c = new lsgd_ctx();
  c->cfg = c0;
  if (alloc && alloc->alloc && alloc->free) {
    c->alloc = *alloc;
    c->have_alloc = true;
  }
  c->stream = (cudaStream_t)cuda_stream;
  c->bf16 = c0.precision == LSGD_BF16;
  c->lsq = m.kind == LSGD_LSQ;
  c->resnet = m.kind == LSGD_RESNET20;
  c->shard = c0.N / c0.K;
  c->T = total_steps_of(c0);
  auto bail = [&](lsgd_status st) {
    if (c->rn) lsgd::resnet_destroy(c->rn);
    free_all(c);
    cudaStreamSynchronize(c->stream);
    cudaGetLastError();
    delete c;
    return st;
  };
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    fail(nullptr, LSGD_ECUDA, "no CUDA device");
    return bail(LSGD_ECUDA);
  }

  const int K = c0.K, B = c0.B_loc;
  if (c->resnet) {
    c->rn = lsgd::resnet_plan_create(c0);
    if (!c->rn) {
      fail(nullptr, LSGD_ENOMEM, "ResNet plan creation failed");
      return bail(LSGD_ENOMEM);
    }
    c->d = lsgd::resnet_num_params(c->rn);
    c->d_pad = lsgd::resnet_d_pad(c->rn);
    lsgd::resnet_segments(c->rn, [&](int64_t canon, int64_t pad, int64_t len) {
      c->segs.push_back({canon, pad, len});
    });
    lsgd::resnet_decay_region(c->rn, &c->wd_period, &c->wd_end);
    c->D = m.in_h * m.in_w * m.in_c;
    c->C = m.n_classes;
  } else {
    build_dense_layout(c);
    c->D = m.widths[0];
    c->C = m.widths[m.n_layers];
  }

  const size_t n_rep = (size_t)K * c->d_pad;
  c->W = (float*)dalloc(c, n_rep * 4);
  c->G = (float*)dalloc(c, n_rep * 4);
  if (c0.momentum != 0.0) c->U = (float*)dalloc(c, n_rep * 4);
  if (c->bf16) c->Wb = (uint16_t*)dalloc(c, n_rep * 2);
  if (!c->bf16 && !c->resnet) {
    c->simt_ws_floats = 1 << 20;
    c->simt_ws = (float*)dalloc(c, (size_t)c->simt_ws_floats * 4);
  }
  c->idx = (int32_t*)dalloc(c, (size_t)K * B * 4);
  c->yb = (int32_t*)dalloc(c, (size_t)K * B * 4);
  c->tb = (float*)dalloc(c, (size_t)K * B * 4);
  c->loss_cap = c->T;
  c->loss_hist = (float*)dalloc(c, (size_t)c->loss_cap * K * 4);
  c->row_loss = (float*)dalloc(c, (size_t)K * B * 4);
  c->flag = (int*)dalloc(c, 16);
  const bool need_ref = c0.compress != LSGD_COMPRESS_NONE || c0.global_momentum > 0.0;
  if (need_ref) {
    c->wref = (float*)dalloc(c, (size_t)c->d_pad * 4);
    c->pnorm = (float*)dalloc(c, (size_t)K * 4);
    c->l1part = (float*)dalloc(c, (size_t)K * lsgd::l1_chunks(c->d_pad) * 4);
    if (c0.compress == LSGD_COMPRESS_EF_SIGN) c->E = (float*)dalloc(c, n_rep * 4);
    if (c0.global_momentum > 0.0) c->ug = (float*)dalloc(c, (size_t)c->d_pad * 4);
    if (!c->wref || !c->pnorm || !c->l1part || (c0.compress == LSGD_COMPRESS_EF_SIGN && !c->E) ||
        (c0.global_momentum > 0.0 && !c->ug)) {
      fail(nullptr, LSGD_ENOMEM, "device allocation failed");
      return bail(LSGD_ENOMEM);
    }
  }
  if (!c->W || !c->G || (c0.momentum != 0.0 && !c->U) || (c->bf16 && !c->Wb) || !c->idx ||
      !c->yb || !c->tb || !c->loss_hist || !c->row_loss || !c->flag) {
    fail(nullptr, LSGD_ENOMEM, "device allocation failed");
    return bail(LSGD_ENOMEM);
  }
  lsgd_status st;
  if (c->resnet) {
    st = lsgd::resnet_alloc(c->rn, [&](size_t bytes) { return dalloc(c, bytes); });
    if (st != LSGD_OK) {
      fail(nullptr, st, "ResNet buffer allocation failed");
      return bail(st);
    }
    st = lsgd::resnet_init_params(c->rn, c->W, c0.seed, c->stream, &c->launches);
  } else {
    st = alloc_dense(c);
    if (st == LSGD_OK) st = init_dense_params(c);
    if (st == LSGD_OK) st = make_tc_maps(c);
    if (st == LSGD_OK && c0.fused_update && c->bf16) {
      c->fused = true;
      for (const DenseLayer& L : c->layers) c->fused = c->fused && L.tc;
    }
    if (st == LSGD_OK) {
      const DenseLayer& top = c->layers.back();
      c->head = c->bf16 && !c->lsq && top.tc && lsgd::head_supported(top.out, c0.B_loc, top.in);
      // A narrow output layer over a long input (the 100-class layer of the 4096-wide MLP) gives
      // the one-tile GEMM only out / 64 x K tiles, each a long reduction that streams from one
      // SM; its forward is split eight ways into partial products that a second kernel adds, in
      // split order, with the bias.
      if (!c->head && !c->lsq && top.tc && top.out <= 128 && top.in >= 1024) {
        const int S = lsgd::tc_valid_splits(top.in, 8);
        if (S > 1) {
          c->logit_parts = (float*)dalloc(c, (size_t)S * c0.K * c0.B_loc * c->ld_logits * 4);
          if (!c->logit_parts) {
            fail(nullptr, LSGD_ENOMEM, "logit partial buffer allocation failed");
            return bail(LSGD_ENOMEM);
          }
          c->logit_splits = S;
        }
      }
      if (defer_top_update(c)) {
        c->dz[2] = dalloc(c, (size_t)c0.K * c0.B_loc * c->ld_dz * 2);
        if (!c->dz[2]) {
          fail(nullptr, LSGD_ENOMEM, "gradient buffer allocation failed");
          return bail(LSGD_ENOMEM);
        }
      }
      // segments averaged outside the weight-gradient + update launches: every bias, and the
      // classifier head's weights when its own kernels update them (each tensor starts at a
      // 64-element boundary, so a length rounded up to 4 stays inside its padding)
      lsgd::AvgSegments& sg = c->avg_segs;
      lsgd::AvgSegments& wg = c->wgrad_segs;
      sg.n = 0;
      wg.n = 0;
      for (size_t l = 0; l < c->layers.size(); ++l) {
        const DenseLayer& Ly = c->layers[l];
        if (c->head && l + 1 == c->layers.size()) {
          sg.off4[sg.n] = Ly.w_off / 4;
          sg.len4[sg.n++] = ((int64_t)Ly.in * Ly.out + 3) / 4;
        } else {
          wg.off4[wg.n] = Ly.w_off / 4;
          wg.len4[wg.n++] = ((int64_t)Ly.in * Ly.out + 3) / 4;
        }
        if (Ly.b_off >= 0) {
          sg.off4[sg.n] = Ly.b_off / 4;
          sg.len4[sg.n++] = ((int64_t)Ly.out + 3) / 4;
        }
      }
    }
  }
  if (st != LSGD_OK) {
    g_last_error = c->err;
    return bail(st);
  }
  if (lsgd::launch_broadcast(c->W, K, c->d_pad, c->stream) != cudaSuccess ||
      (c->bf16 && lsgd::launch_to_bf16(c->W, c->Wb, (int64_t)n_rep, c->stream) != cudaSuccess)) {
    fail(nullptr, LSGD_ECUDA, "initial broadcast failed");
    return bail(LSGD_ECUDA);
  }
  c->launches += c->bf16 ? 2 : 1;
  if (c->wref &&
      cudaMemcpyAsync(c->wref, c->W, (size_t)c->d_pad * 4, cudaMemcpyDeviceToDevice, c->stream) !=
          cudaSuccess) {
    fail(nullptr, LSGD_ECUDA, "initial round-start model copy failed");
    return bail(LSGD_ECUDA);
  }
  cudaError_t e = cudaStreamSynchronize(c->stream);
  if (e != cudaSuccess) {
    fail_cuda(nullptr, e, "lsgd_create");
    return bail(LSGD_ECUDA);
  }
  *out = c;
  return LSGD_OK;
}

void lsgd_destroy(lsgd_ctx* c) {
  if (!c) return;
  if (c->copy_stream) cudaStreamSynchronize(c->copy_stream);
  cudaStreamSynchronize(c->stream);
  for (cudaEvent_t e : c->prof_pool) cudaEventDestroy(e);
  for (int i = 0; i < 2; ++i) {
    if (c->stage_copied[i]) cudaEventDestroy(c->stage_copied[i]);
    if (c->stage_free[i]) cudaEventDestroy(c->stage_free[i]);
  }
  if (c->copy_stream) cudaStreamDestroy(c->copy_stream);
  if (c->rn) lsgd::resnet_destroy(c->rn);
  free_all(c);
  cudaStreamSynchronize(c->stream);
  delete c;
}

static lsgd_status set_data(lsgd_ctx* c, const float* X, const int32_t* labels, const float* targets,
                            int64_t N) {
  if (!c || !X) return fail(c, LSGD_EINVAL, "NULL argument");
  if (N != c->cfg.N) return fail(c, LSGD_EINVAL, "N differs from the configured dataset size");
  if (c->lsq != (targets != nullptr) || (!c->lsq && !labels))
    return fail(c, LSGD_EINVAL, "labels for classifiers, targets for least squares");
  if (labels)
    for (int64_t i = 0; i < N; ++i)
      if (labels[i] < 0 || labels[i] >= c->C) return fail(c, LSGD_EINVAL, "label out of range");
  if (!c->X) {
    c->X = (float*)dalloc(c, (size_t)N * c->D * 4);
    if (!c->X) return fail(c, LSGD_ENOMEM, "dataset allocation failed");
    if (labels) c->y = (int32_t*)dalloc(c, (size_t)N * 4);
    if (targets) c->t = (float*)dalloc(c, (size_t)N * 4);
    if ((labels && !c->y) || (targets && !c->t)) return fail(c, LSGD_ENOMEM, "label allocation failed");
  }
  LSGD_TRY_CUDA(c, cudaMemcpyAsync(c->X, X, (size_t)N * c->D * 4, cudaMemcpyHostToDevice, c->stream));
  if (labels)
    LSGD_TRY_CUDA(c, cudaMemcpyAsync(c->y, labels, (size_t)N * 4, cudaMemcpyHostToDevice, c->stream));
  if (targets)
    LSGD_TRY_CUDA(c, cudaMemcpyAsync(c->t, targets, (size_t)N * 4, cudaMemcpyHostToDevice, c->stream));
  LSGD_TRY_CUDA(c, cudaStreamSynchronize(c->stream));
  c->have_data = true;
  return LSGD_OK;
}

lsgd_status lsgd_set_dataset(lsgd_ctx* c, const float* X, const int32_t* labels, int64_t N) {
  if (c && c->lsq) return fail(c, LSGD_EINVAL, "least squares takes lsgd_set_targets");
  return set_data(c, X, labels, nullptr, N);
}

lsgd_status lsgd_set_targets(lsgd_ctx* c, const float* X, const float* targets, int64_t N) {
  if (c && !c->lsq) return fail(c, LSGD_EINVAL, "targets are for least squares only");
  return set_data(c, X, nullptr, targets, N);
}

static lsgd_status local_step(lsgd_ctx* c, bool avg) {
  if (!c) return fail(nullptr, LSGD_EINVAL, "NULL context");
  if (!c->have_data) return fail(c, LSGD_ESTATE, "lsgd_set_dataset must come first");
  const int K = c->cfg.K, B = c->cfg.B_loc;
  const int64_t e0 = prof_mark(c);
  LSGD_LAUNCH(c, lsgd::launch_sample_indices(c->idx, c->cfg.seed, c->step, K, B, c->cfg.N,
                                             c->cfg.sampling, c->stream));
  LSGD_LAUNCH(c, lsgd::launch_gather_rows(input_buffer(c), c->bf16, input_ld(c), c->X, c->D, c->idx,
                                          K * B, c->y, c->y ? c->yb : nullptr, c->t,
                                          c->t ? c->tb : nullptr, c->stream));
  return step_body(c, e0, avg);
}

lsgd_status lsgd_local_step(lsgd_ctx* c) { return local_step(c, false); }

static lsgd_status local_step_batch(lsgd_ctx* c, const float* x, const void* lab, int on_device,
                                    bool avg) {
  if (!c || !x || !lab) return fail(c, LSGD_EINVAL, "NULL argument");
  const int K = c->cfg.K, B = c->cfg.B_loc;
  const size_t rows = (size_t)K * B;
  const float* xs = x;
  const void* ls = lab;
  const int64_t e0 = prof_mark(c);
  int sl = -1;
  if (!on_device) {
    // staging buffer sl: its copy waits until the gather of two batches ago has read it, and this
    // step's gather waits for the copy; nothing else orders the copy stream against the step
    if (!c->copy_stream) {
      LSGD_TRY_CUDA(c, cudaStreamCreateWithFlags(&c->copy_stream, cudaStreamNonBlocking));
      for (int i = 0; i < 2; ++i) {
        LSGD_TRY_CUDA(c, cudaEventCreateWithFlags(&c->stage_copied[i], cudaEventDisableTiming));
        LSGD_TRY_CUDA(c, cudaEventCreateWithFlags(&c->stage_free[i], cudaEventDisableTiming));
      }
    }
    sl = c->stage_next;
    if (!c->xstage[sl]) {
      c->xstage[sl] = (float*)dalloc(c, rows * c->D * 4);
      c->lstage[sl] = dalloc(c, rows * 4);
      if (!c->xstage[sl] || !c->lstage[sl]) return fail(c, LSGD_ENOMEM, "staging allocation failed");
    }
    if (c->stage_used[sl]) LSGD_TRY_CUDA(c, cudaStreamWaitEvent(c->copy_stream, c->stage_free[sl], 0));
    LSGD_TRY_CUDA(c, cudaMemcpyAsync(c->xstage[sl], x, rows * c->D * 4, cudaMemcpyHostToDevice,
                                     c->copy_stream));
    LSGD_TRY_CUDA(c, cudaMemcpyAsync(c->lstage[sl], lab, rows * 4, cudaMemcpyHostToDevice,
                                     c->copy_stream));
    LSGD_TRY_CUDA(c, cudaEventRecord(c->stage_copied[sl], c->copy_stream));
    LSGD_TRY_CUDA(c, cudaStreamWaitEvent(c->stream, c->stage_copied[sl], 0));
    c->stage_next ^= 1;
    xs = c->xstage[sl];
    ls = c->lstage[sl];
  }
  const int32_t* yl = c->lsq ? nullptr : (const int32_t*)ls;
  const float* tl = c->lsq ? (const float*)ls : nullptr;
  LSGD_LAUNCH(c, lsgd::launch_gather_rows(input_buffer(c), c->bf16, input_ld(c), xs, c->D, nullptr,
                                          (int)rows, yl, yl ? c->yb : nullptr, tl,
                                          tl ? c->tb : nullptr, c->stream));
  if (sl >= 0) {
    LSGD_TRY_CUDA(c, cudaEventRecord(c->stage_free[sl], c->stream));
    c->stage_used[sl] = true;
  }
  return step_body(c, e0, avg);
}

lsgd_status lsgd_local_step_batch(lsgd_ctx* c, const float* x, const void* lab, int on_device) {
  return local_step_batch(c, x, lab, on_device, false);
}

lsgd_status lsgd_sync_average(lsgd_ctx* c) {
  if (!c) return fail(nullptr, LSGD_EINVAL, "NULL context");
  if (lsgd_status st = materialize(c); st != LSGD_OK) return st;
  const int64_t e0 = prof_mark(c);
  const int K = c->cfg.K;
  if (c->cfg.compress != LSGD_COMPRESS_NONE) {
    // Algorithms 4 / 5: sign-compressed model differences relative to the round start
    LSGD_LAUNCH(c, lsgd::launch_l1_norms(c->W, c->wref, c->E, K, c->d_pad, c->d, c->l1part, c->pnorm,
                                         c->stream));
    c->launches++;  // launch_l1_norms runs two kernels (chunk sums, then their total)
    LSGD_LAUNCH(c, lsgd::launch_sign_sync(c->W, c->Wb, c->wref, c->E, c->pnorm, K, c->d_pad, c->stream));
  } else if (c->cfg.global_momentum > 0.0) {
    // Sec. C.3.1 global momentum with the step size of the step that ended the round
    const float lr = (float)lr_at(c->cfg, c->T, c->step > 0 ? c->step - 1 : 0);
    LSGD_LAUNCH(c, lsgd::launch_gm_sync(c->W, c->Wb, c->wref, c->ug, K, c->d_pad, lr,
                                        (float)c->cfg.global_momentum, c->stream));
  } else {
    LSGD_LAUNCH(c, lsgd::launch_kway_average(c->W, c->Wb, K, c->d_pad, c->stream));
  }
  prof_span(c, LSGD_PH_AVERAGE, e0, prof_mark(c));
  c->syncs++;
  c->synced = true;  // every variant leaves all replicas at one model
  return LSGD_OK;
}

lsgd_status lsgd_block_average(lsgd_ctx* c) {
  if (!c) return fail(nullptr, LSGD_EINVAL, "NULL context");
  if (c->cfg.hier_block <= 0) return fail(c, LSGD_ESTATE, "the context has no averaging blocks");
  if (lsgd_status st = materialize(c); st != LSGD_OK) return st;
  const int64_t e0 = prof_mark(c);
  LSGD_LAUNCH(c, lsgd::launch_group_average(c->W, c->Wb, c->cfg.hier_block,
                                            c->cfg.K / c->cfg.hier_block, c->d_pad, c->stream));
  prof_span(c, LSGD_PH_AVERAGE, e0, prof_mark(c));
  c->block_syncs++;
  c->synced = c->cfg.hier_block >= c->cfg.K;
  return LSGD_OK;
}

lsgd_status lsgd_profile_enable(lsgd_ctx* c, int enable) {
  if (!c) return fail(nullptr, LSGD_EINVAL, "NULL context");
  LSGD_TRY_CUDA(c, cudaStreamSynchronize(c->stream));
  c->prof_spans.clear();
  c->prof_used = 0;
  c->prof_on = enable != 0;
  return LSGD_OK;
}

lsgd_status lsgd_profile_read(lsgd_ctx* c, lsgd_profile* out) {
  if (!c || !out) return fail(c, LSGD_EINVAL, "NULL argument");
  LSGD_TRY_CUDA(c, cudaStreamSynchronize(c->stream));
  lsgd_profile p{};
  for (const auto& sp : c->prof_spans) {
    float ms = 0.f;
    LSGD_TRY_CUDA(c, cudaEventElapsedTime(&ms, c->prof_pool[sp[1]], c->prof_pool[sp[2]]));
    p.count[sp[0]]++;
    p.ms[sp[0]] += ms;
  }
  *out = p;
  return LSGD_OK;
}

lsgd_status lsgd_run(lsgd_ctx* c, int64_t n_steps) {
  if (!c) return fail(nullptr, LSGD_EINVAL, "NULL context");
  if (n_steps < 0) return fail(c, LSGD_EINVAL, "n_steps must be >= 0");
  for (int64_t i = 0; i < n_steps; ++i) {
    const int kind = sync_kind_at(c->cfg, c->T, c->step, &c->cursor);
    if (kind == 2 && can_fuse_average(c)) {
      // the step's update launches also form the K-way average
      lsgd_status st = local_step(c, true);
      if (st != LSGD_OK) return st;
      continue;
    }
    lsgd_status st = lsgd_local_step(c);
    if (st != LSGD_OK) return st;
    if (kind == 2) {
      st = lsgd_sync_average(c);
      if (st != LSGD_OK) return st;
    } else if (kind == 1) {
      st = lsgd_block_average(c);
      if (st != LSGD_OK) return st;
    }
  }
  return LSGD_OK;
}

lsgd_status lsgd_run_batch(lsgd_ctx* c, const float* x, const void* labels_or_targets,
                           int on_device) {
  if (!c) return fail(nullptr, LSGD_EINVAL, "NULL context");
  const int kind = sync_kind_at(c->cfg, c->T, c->step, &c->cursor);
  const bool fuse = kind == 2 && can_fuse_average(c);
  lsgd_status st = local_step_batch(c, x, labels_or_targets, on_device, fuse);
  if (st != LSGD_OK || fuse) return st;
  if (kind == 2) return lsgd_sync_average(c);
  if (kind == 1) return lsgd_block_average(c);
  return LSGD_OK;
}

static lsgd_status get_vec(lsgd_ctx* c, const float* buf, int k, float* dst, int dst_is_device,
                           size_t n) {
  if (!c || !dst) return fail(c, LSGD_EINVAL, "NULL argument");
  if (n != (size_t)c->d) return fail(c, LSGD_EINVAL, "n must equal lsgd_num_params()");
  if (k < -1 || k >= c->cfg.K) return fail(c, LSGD_EINVAL, "replica index out of range");
  if (lsgd_status st = materialize(c); st != LSGD_OK) return st;
  if (!buf) {  // no momentum buffer: momentum is identically zero
    if (dst_is_device)
      LSGD_TRY_CUDA(c, cudaMemsetAsync(dst, 0, n * 4, c->stream));
    else
      std::memset(dst, 0, n * 4);
    LSGD_TRY_CUDA(c, cudaStreamSynchronize(c->stream));
    return LSGD_OK;
  }
  if (k >= 0) {
    const cudaMemcpyKind kind = dst_is_device ? cudaMemcpyDeviceToDevice : cudaMemcpyDeviceToHost;
    for (const Seg& s : c->segs)
      LSGD_TRY_CUDA(c, cudaMemcpyAsync(dst + s.canon, buf + (int64_t)k * c->d_pad + s.pad,
                                       (size_t)s.len * 4, kind, c->stream));
    LSGD_TRY_CUDA(c, cudaStreamSynchronize(c->stream));
    return LSGD_OK;
  }
  std::vector<float> all((size_t)c->cfg.K * c->d_pad);
  LSGD_TRY_CUDA(c, cudaMemcpyAsync(all.data(), buf, all.size() * 4, cudaMemcpyDeviceToHost, c->stream));
  LSGD_TRY_CUDA(c, cudaStreamSynchronize(c->stream));
  std::vector<float> mean((size_t)c->d);
  for (const Seg& s : c->segs)
    for (int64_t i = 0; i < s.len; ++i) {
      double acc = 0.0;
      for (int kk = 0; kk < c->cfg.K; ++kk) acc += all[(size_t)kk * c->d_pad + s.pad + i];
      mean[s.canon + i] = (float)(acc / c->cfg.K);
    }
  if (dst_is_device) {
    LSGD_TRY_CUDA(c, cudaMemcpyAsync(dst, mean.data(), n * 4, cudaMemcpyHostToDevice, c->stream));
    LSGD_TRY_CUDA(c, cudaStreamSynchronize(c->stream));
  } else {
    std::memcpy(dst, mean.data(), n * 4);
  }
  return LSGD_OK;
}

lsgd_status lsgd_params(lsgd_ctx* c, int k, float* dst, int dst_is_device, size_t n) {
  return get_vec(c, c ? c->W : nullptr, k, dst, dst_is_device, n);
}

lsgd_status lsgd_momentum(lsgd_ctx* c, int k, float* dst, int dst_is_device, size_t n) {
  return get_vec(c, c ? c->U : nullptr, k, dst, dst_is_device, n);
}

static lsgd_status set_vec(lsgd_ctx* c, float* buf, int k, const float* src, size_t n, bool is_w) {
  if (!c || !src) return fail(c, LSGD_EINVAL, "NULL argument");
  if (n != (size_t)c->d) return fail(c, LSGD_EINVAL, "n must equal lsgd_num_params()");
  if (k < -1 || k >= c->cfg.K) return fail(c, LSGD_EINVAL, "replica index out of range");
  if (!buf) return fail(c, LSGD_ESTATE, "no momentum buffer (momentum is 0)");
  if (lsgd_status st = materialize(c); st != LSGD_OK) return st;
  const int k0 = k < 0 ? 0 : k;
  for (const Seg& s : c->segs)
    LSGD_TRY_CUDA(c, cudaMemcpyAsync(buf + (int64_t)k0 * c->d_pad + s.pad, src + s.canon,
                                     (size_t)s.len * 4, cudaMemcpyHostToDevice, c->stream));
  if (k < 0) LSGD_LAUNCH(c, lsgd::launch_broadcast(buf, c->cfg.K, c->d_pad, c->stream));
  if (is_w && k < 0 && c->wref)
    LSGD_TRY_CUDA(c, cudaMemcpyAsync(c->wref, c->W, (size_t)c->d_pad * 4, cudaMemcpyDeviceToDevice,
                                     c->stream));
  if (is_w && c->Wb)
    LSGD_LAUNCH(c, lsgd::launch_to_bf16(c->W, c->Wb, (int64_t)c->cfg.K * c->d_pad, c->stream));
  if (is_w) c->synced = k < 0 || c->cfg.K == 1;
  LSGD_TRY_CUDA(c, cudaStreamSynchronize(c->stream));
  return LSGD_OK;
}

lsgd_status lsgd_set_params(lsgd_ctx* c, int k, const float* src, size_t n) {
  return set_vec(c, c ? c->W : nullptr, k, src, n, true);
}

lsgd_status lsgd_set_momentum(lsgd_ctx* c, int k, const float* src, size_t n) {
  return set_vec(c, c ? c->U : nullptr, k, src, n, false);
}

// The arrays behind lsgd_sync_state: the replica stride is d_pad for E and 0 for the others.
static float* sync_state_buf(lsgd_ctx* c, int which, bool* per_replica) {
  *per_replica = which == LSGD_STATE_ERROR;
  switch (which) {
    case LSGD_STATE_WREF: return c->wref;
    case LSGD_STATE_ERROR: return c->E;
    case LSGD_STATE_GLOBAL_MOMENTUM: return c->ug;
    default: return nullptr;
  }
}

lsgd_status lsgd_sync_state(lsgd_ctx* c, int which, int k, float* dst, size_t n) {
  if (!c || !dst) return fail(c, LSGD_EINVAL, "NULL argument");
  if (n != (size_t)c->d) return fail(c, LSGD_EINVAL, "n must equal lsgd_num_params()");
  bool per = false;
  float* buf = sync_state_buf(c, which, &per);
  if (!buf) return fail(c, LSGD_ESTATE, "this configuration keeps no such synchronisation state");
  if (per ? (k < 0 || k >= c->cfg.K) : k != 0)
    return fail(c, LSGD_EINVAL, "replica index out of range for this state");
  for (const Seg& s : c->segs)
    LSGD_TRY_CUDA(c, cudaMemcpyAsync(dst + s.canon, buf + (int64_t)k * c->d_pad + s.pad,
                                     (size_t)s.len * 4, cudaMemcpyDeviceToHost, c->stream));
  LSGD_TRY_CUDA(c, cudaStreamSynchronize(c->stream));
  return LSGD_OK;
}

lsgd_status lsgd_set_sync_state(lsgd_ctx* c, int which, int k, const float* src, size_t n) {
  if (!c || !src) return fail(c, LSGD_EINVAL, "NULL argument");
  if (n != (size_t)c->d) return fail(c, LSGD_EINVAL, "n must equal lsgd_num_params()");
  bool per = false;
  float* buf = sync_state_buf(c, which, &per);
  if (!buf) return fail(c, LSGD_ESTATE, "this configuration keeps no such synchronisation state");
  if (per ? (k < -1 || k >= c->cfg.K) : k != 0)
    return fail(c, LSGD_EINVAL, "replica index out of range for this state");
  const int k0 = k < 0 ? 0 : k;
  for (const Seg& s : c->segs)
    LSGD_TRY_CUDA(c, cudaMemcpyAsync(buf + (int64_t)k0 * c->d_pad + s.pad, src + s.canon,
                                     (size_t)s.len * 4, cudaMemcpyHostToDevice, c->stream));
  if (per && k < 0) LSGD_LAUNCH(c, lsgd::launch_broadcast(buf, c->cfg.K, c->d_pad, c->stream));
  LSGD_TRY_CUDA(c, cudaStreamSynchronize(c->stream));
  return LSGD_OK;
}

static lsgd_status copy_losses(lsgd_ctx* c, float* dst, int64_t n_steps) {
  if (!c || !dst) return fail(c, LSGD_EINVAL, "NULL argument");
  if (n_steps < 0 || n_steps > c->step || n_steps > c->loss_cap)
    return fail(c, LSGD_EINVAL, "n_steps exceeds the recorded history");
  const int K = c->cfg.K;
  for (int64_t i = 0; i < n_steps; ++i) {
    const int64_t s = c->step - n_steps + i;
    LSGD_TRY_CUDA(c, cudaMemcpyAsync(dst + i * K, c->loss_hist + (s % c->loss_cap) * K, (size_t)K * 4,
                                     cudaMemcpyDeviceToHost, c->stream));
  }
  return LSGD_OK;
}

lsgd_status lsgd_losses(lsgd_ctx* c, float* dst, int64_t n_steps) {
  lsgd_status st = copy_losses(c, dst, n_steps);
  if (st != LSGD_OK) return st;
  LSGD_TRY_CUDA(c, cudaStreamSynchronize(c->stream));
  return LSGD_OK;
}

lsgd_status lsgd_losses_async(lsgd_ctx* c, float* dst, int64_t n_steps) {
  return copy_losses(c, dst, n_steps);
}

lsgd_status lsgd_synchronize(lsgd_ctx* c) {
  if (!c) return fail(nullptr, LSGD_EINVAL, "NULL context");
  if (c->copy_stream) LSGD_TRY_CUDA(c, cudaStreamSynchronize(c->copy_stream));
  LSGD_TRY_CUDA(c, cudaStreamSynchronize(c->stream));
  return LSGD_OK;
}

lsgd_status lsgd_debug_indices(lsgd_ctx* c, int64_t step, int32_t* dst) {
  if (!c || !dst) return fail(c, LSGD_EINVAL, "NULL argument");
  if (step < 0) return fail(c, LSGD_EINVAL, "step must be >= 0");
  const int K = c->cfg.K, B = c->cfg.B_loc;
  int32_t* tmp = (int32_t*)dalloc(c, (size_t)K * B * 4);
  if (!tmp) return fail(c, LSGD_ENOMEM, "scratch allocation failed");
  cudaError_t e =
      lsgd::launch_sample_indices(tmp, c->cfg.seed, step, K, B, c->cfg.N, c->cfg.sampling, c->stream);
  c->launches++;
  if (e == cudaSuccess) e = cudaMemcpyAsync(dst, tmp, (size_t)K * B * 4, cudaMemcpyDeviceToHost, c->stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
  // release the scratch buffer
  c->allocs.pop_back();
  if (c->have_alloc)
    c->alloc.free(c->alloc.user, tmp, (void*)c->stream);
  else
    cudaFreeAsync(tmp, c->stream);
  if (e != cudaSuccess) return fail_cuda(c, e, "lsgd_debug_indices");
  return LSGD_OK;
}

lsgd_status lsgd_eval_loss(lsgd_ctx* c, int k, int64_t n, double* loss) {
  if (!c || !loss) return fail(c, LSGD_EINVAL, "NULL argument");
  if (!c->have_data) return fail(c, LSGD_ESTATE, "lsgd_set_dataset must come first");
  if (k < -1 || k >= c->cfg.K) return fail(c, LSGD_EINVAL, "replica index out of range");
  if (n < 1 || n > c->cfg.N) return fail(c, LSGD_EINVAL, "n must be in [1, N]");
  if (lsgd_status st = materialize(c); st != LSGD_OK) return st;
  const int kk = k < 0 ? 0 : k;
  const int K = c->cfg.K, B = c->cfg.B_loc;
  const int64_t per = (int64_t)K * B;
  std::vector<float> rl((size_t)per);
  double total = 0.0;
  for (int64_t start = 0; start < n; start += per) {
    const int rows = (int)std::min<int64_t>(per, n - start);
    LSGD_LAUNCH(c, lsgd::launch_gather_rows(input_buffer(c), c->bf16, input_ld(c), c->X + start * c->D,
                                            c->D, nullptr, rows, c->y ? c->y + start : nullptr,
                                            c->y ? c->yb : nullptr, c->t ? c->t + start : nullptr,
                                            c->t ? c->tb : nullptr, c->stream));
    const int groups = (rows + B - 1) / B;
    lsgd_status st;
    if (c->resnet) {
      st = lsgd::resnet_eval(c->rn, c->W, c->Wb, c->d_pad, kk, groups, c->yb, c->row_loss, c->stream,
                             &c->launches);
      if (st != LSGD_OK) return fail(c, st, lsgd::resnet_last_error(c->rn));
    } else {
      st = dense_forward(c, groups, kk, 0);
      if (st != LSGD_OK) return st;
      st = dense_loss(c, groups, true, nullptr);
      if (st != LSGD_OK) return st;
    }
    LSGD_TRY_CUDA(c, cudaMemcpyAsync(rl.data(), c->row_loss, (size_t)rows * 4, cudaMemcpyDeviceToHost,
                                     c->stream));
    LSGD_TRY_CUDA(c, cudaStreamSynchronize(c->stream));
    for (int r = 0; r < rows; ++r) total += rl[r];
  }
  *loss = total / (double)n;
  return LSGD_OK;
}

lsgd_status lsgd_device_status(lsgd_ctx* c) {
  if (c) LSGD_TRY_CUDA(c, cudaStreamSynchronize(c->stream));
  if (lsgd::tc_take_timeout_flag())
    return fail(c, LSGD_ETIMEOUT,
                "a bounded wait inside a tensor-core kernel ran out; results since the last check "
                "are not valid");
  return LSGD_OK;
}

lsgd_status lsgd_bounded_wait_selftest(int arrive, double limit_ms, void* stream) {
  if (!(limit_ms >= 0.0) || limit_ms > 1000.0)
    return fail(nullptr, LSGD_EINVAL, "limit_ms must be in [0, 1000]");
  int dev = 0, khz = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&khz, cudaDevAttrClockRate, dev) != cudaSuccess || khz <= 0) {
    cudaGetLastError();
    return fail(nullptr, LSGD_ECUDA, "cannot read the SM clock rate");
  }
  const cudaStream_t st = (cudaStream_t)stream;
  const long long cycles = (long long)(limit_ms * (double)khz);
  int* d_out = nullptr;
  int h_out = -1;
  cudaError_t e = cudaMallocAsync((void**)&d_out, sizeof(int), st);
  if (e == cudaSuccess) e = lsgd::launch_bounded_wait_selftest(cycles, arrive, d_out, st);
  if (e == cudaSuccess) e = cudaMemcpyAsync(&h_out, d_out, sizeof(int), cudaMemcpyDeviceToHost, st);
  if (d_out) cudaFreeAsync(d_out, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return fail_cuda(nullptr, e, "lsgd_bounded_wait_selftest");
  const int flagged = lsgd::tc_take_timeout_flag();
  if (h_out == 1 && !flagged) return LSGD_OK;
  if (h_out == 0 && flagged) return fail(nullptr, LSGD_ETIMEOUT, "bounded wait ran out (as asked)");
  return fail(nullptr, LSGD_ECUDA, "bounded-wait self-test: inconsistent result");
}

lsgd_status lsgd_check_finite(lsgd_ctx* c) {
  if (!c) return fail(nullptr, LSGD_EINVAL, "NULL context");
  const lsgd_status ds = lsgd_device_status(c);
  if (ds != LSGD_OK) return ds;
  if (lsgd_status st = materialize(c); st != LSGD_OK) return st;
  LSGD_TRY_CUDA(c, cudaMemsetAsync(c->flag, 0, 4, c->stream));
  LSGD_LAUNCH(c, lsgd::launch_check_finite(c->W, (int64_t)c->cfg.K * c->d_pad, c->flag, c->stream));
  int h = 0;
  LSGD_TRY_CUDA(c, cudaMemcpyAsync(&h, c->flag, 4, cudaMemcpyDeviceToHost, c->stream));
  LSGD_TRY_CUDA(c, cudaStreamSynchronize(c->stream));
  if (h) return fail(c, LSGD_ENONFINITE, "non-finite parameter found");
  return LSGD_OK;
}

static const uint64_t kMagic = 0x3330545043445347ULL;  // "GSDCPT03"

// Bit mask of the state arrays a checkpoint holds after W: 1 momentum, 2 round-start model,
// 4 error-feedback memories, 8 global momentum.  A checkpoint loads only into a context that
// keeps exactly the same arrays.
static int64_t state_mask(const lsgd_ctx* c) {
  return (c->U ? 1 : 0) | (c->wref ? 2 : 0) | (c->E ? 4 : 0) | (c->ug ? 8 : 0);
}

lsgd_status lsgd_save(lsgd_ctx* c, const char* path) {
  if (!c || !path) return fail(c, LSGD_EINVAL, "NULL argument");
  if (lsgd_status st = materialize(c); st != LSGD_OK) return st;
  const size_t n = (size_t)c->cfg.K * c->d_pad;
  std::vector<float> buf(n);
  FILE* f = std::fopen(path, "wb");
  if (!f) return fail(c, LSGD_EIO, std::string("cannot open ") + path);
  int64_t hdr[7] = {(int64_t)kMagic, c->cfg.K, c->d_pad, c->step, c->syncs, state_mask(c),
                    c->block_syncs};
  bool ok = std::fwrite(hdr, sizeof(hdr), 1, f) == 1;
  // w and u of every replica, then the synchronisation state the context keeps
  std::vector<std::pair<const float*, size_t>> parts = {{c->W, n}};
  if (c->U) parts.push_back({c->U, n});
  if (c->wref) parts.push_back({c->wref, (size_t)c->d_pad});
  if (c->E) parts.push_back({c->E, n});
  if (c->ug) parts.push_back({c->ug, (size_t)c->d_pad});
  for (size_t which = 0; ok && which < parts.size(); ++which) {
    const float* src = parts[which].first;
    const size_t cnt = parts[which].second;
    cudaError_t e = cudaMemcpyAsync(buf.data(), src, cnt * 4, cudaMemcpyDeviceToHost, c->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
    if (e != cudaSuccess) {
      std::fclose(f);
      return fail_cuda(c, e, "lsgd_save");
    }
    ok = std::fwrite(buf.data(), 4, cnt, f) == cnt;
  }
  ok = (std::fclose(f) == 0) && ok;
  if (!ok) return fail(c, LSGD_EIO, "write failed");
  return LSGD_OK;
}

lsgd_status lsgd_load(lsgd_ctx* c, const char* path) {
  if (!c || !path) return fail(c, LSGD_EINVAL, "NULL argument");
  if (lsgd_status st = materialize(c); st != LSGD_OK) return st;  // a failed load keeps the state
  FILE* f = std::fopen(path, "rb");
  if (!f) return fail(c, LSGD_EIO, std::string("cannot open ") + path);
  int64_t hdr[7];
  if (std::fread(hdr, sizeof(hdr), 1, f) != 1 || hdr[0] != (int64_t)kMagic || hdr[1] != c->cfg.K ||
      hdr[2] != c->d_pad || hdr[5] != state_mask(c)) {
    std::fclose(f);
    return fail(c, LSGD_EIO, "checkpoint does not match this configuration");
  }
  const size_t n = (size_t)c->cfg.K * c->d_pad;
  std::vector<float> buf(n);
  std::vector<std::pair<float*, size_t>> parts = {{c->W, n}};
  if (c->U) parts.push_back({c->U, n});
  if (c->wref) parts.push_back({c->wref, (size_t)c->d_pad});
  if (c->E) parts.push_back({c->E, n});
  if (c->ug) parts.push_back({c->ug, (size_t)c->d_pad});
  for (size_t which = 0; which < parts.size(); ++which) {
    float* dst = parts[which].first;
    const size_t cnt = parts[which].second;
    if (std::fread(buf.data(), 4, cnt, f) != cnt) {
      std::fclose(f);
      return fail(c, LSGD_EIO, "truncated checkpoint");
    }
    cudaError_t e = cudaMemcpyAsync(dst, buf.data(), cnt * 4, cudaMemcpyHostToDevice, c->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
    if (e != cudaSuccess) {
      std::fclose(f);
      return fail_cuda(c, e, "lsgd_load");
    }
  }
  std::fclose(f);
  if (c->Wb) LSGD_LAUNCH(c, lsgd::launch_to_bf16(c->W, c->Wb, (int64_t)n, c->stream));
  LSGD_TRY_CUDA(c, cudaStreamSynchronize(c->stream));
  c->step = hdr[3];
  c->syncs = hdr[4];
  c->block_syncs = hdr[6];
  c->synced = c->cfg.K == 1;  // the file does not say whether the replicas agree
  return LSGD_OK;
}

int64_t lsgd_num_params(const lsgd_ctx* c) { return c ? c->d : -1; }
int64_t lsgd_step_count(const lsgd_ctx* c) { return c ? c->step : -1; }

lsgd_status lsgd_set_step(lsgd_ctx* c, int64_t step) {
  if (!c) return fail(nullptr, LSGD_EINVAL, "NULL context");
  if (step < 0 || step > c->T) return fail(c, LSGD_EINVAL, "step must lie in [0, T]");
  c->step = step;  // steps already enqueued carry their own s, learning rate and sync kind
  c->cursor = RoundCursor{};
  return LSGD_OK;
}
int64_t lsgd_sync_count(const lsgd_ctx* c) { return c ? c->syncs : -1; }
int64_t lsgd_block_sync_count(const lsgd_ctx* c) { return c ? c->block_syncs : -1; }
lsgd_status lsgd_schedule(const lsgd_config* cfg, int64_t n_steps, double* lr, int32_t* sync_kind) {
  if (!cfg || n_steps < 0) return fail(nullptr, LSGD_EINVAL, "lsgd_schedule: bad arguments");
  const lsgd_status st = validate_config(*cfg);
  if (st != LSGD_OK) return st;
  const int64_t T = total_steps_of(*cfg);
  RoundCursor cur;
  for (int64_t s = 0; s < n_steps; ++s) {
    if (lr) lr[s] = lr_at(*cfg, T, s);
    if (sync_kind) sync_kind[s] = sync_kind_at(*cfg, T, s, &cur);
  }
  return LSGD_OK;
}

int64_t lsgd_total_steps(const lsgd_ctx* c) { return c ? c->T : -1; }
double lsgd_lr_at(const lsgd_ctx* c, int64_t s) { return c ? lr_at(c->cfg, c->T, s) : 0.0; }
int64_t lsgd_kernel_launches(const lsgd_ctx* c) { return c ? c->launches : -1; }

const char* lsgd_last_error(const lsgd_ctx* c) {
  if (c) return c->err.c_str();
  return g_last_error.c_str();
}

// ---- stand-alone kernels ----
lsgd_status lsgd_kway_average(float* W, uint16_t* Wb, int K, int64_t d, void* stream) {
  if (!W || K < 1 || d < 0 || (d & 3) || ((uintptr_t)W & 15) || ((uintptr_t)Wb & 7))
    return fail(nullptr, LSGD_EINVAL, "lsgd_kway_average: bad arguments");
  cudaError_t e = lsgd::launch_kway_average(W, Wb, K, d, (cudaStream_t)stream);
  if (e != cudaSuccess) return fail_cuda(nullptr, e, "lsgd_kway_average");
  return LSGD_OK;
}

lsgd_status lsgd_sgd_update(float* w, float* u, const float* g, uint16_t* Wb, int64_t n, float lr,
                            float momentum, int nesterov, float weight_decay, int64_t period,
                            int64_t decay_end, void* stream) {
  if (!w || !g || n < 0 || (n & 3) || (period & 3) || (decay_end & 3) || ((uintptr_t)w & 15) ||
      ((uintptr_t)g & 15) || ((uintptr_t)u & 15) || ((uintptr_t)Wb & 7) || (momentum != 0.f && !u))
    return fail(nullptr, LSGD_EINVAL, "lsgd_sgd_update: bad arguments");
  cudaError_t e = lsgd::launch_sgd_update(w, u, g, Wb, n, lr, momentum, nesterov, weight_decay, period,
                                          decay_end, (cudaStream_t)stream);
  if (e != cudaSuccess) return fail_cuda(nullptr, e, "lsgd_sgd_update");
  return LSGD_OK;
}

lsgd_status lsgd_grouped_gemm_bf16(const uint16_t* A, int a_mn, const uint16_t* B, int b_mn, float* C,
                                   int M, int N, int Kd, int G, int engine, void* stream) {
  if (!A || !B || !C || M < 1 || N < 1 || Kd < 1 || G < 1 || G > 65535 || (engine != 0 && engine != 1))
    return fail(nullptr, LSGD_EINVAL, "lsgd_grouped_gemm_bf16: bad arguments");
  const int a_inner = a_mn ? M : Kd, b_inner = b_mn ? N : Kd;
  if ((a_inner % 8) || (b_inner % 8) || ((uintptr_t)A & 15) || ((uintptr_t)B & 15) || ((uintptr_t)C & 15))
    return fail(nullptr, LSGD_EINVAL, "lsgd_grouped_gemm_bf16: contiguous extents must be multiples of 8");
  cudaStream_t s = (cudaStream_t)stream;
  cudaError_t e;
  if (engine == 0) {
    if (!lsgd::tc_available()) return fail(nullptr, LSGD_EUNSUPPORTED, "tcgen05 not available");
    lsgd::TcGemmArgs t{};
    t.M = M;
    t.N = N;
    t.Kd = Kd;
    t.G = G;
    bool ok;
    if (a_mn) {
      ok = lsgd::make_tma_map_bf16(&t.A.map, A, M, Kd, G, M, (uint64_t)M * Kd, 64, 64);
      t.A.box_rows = 64;
    } else {
      ok = lsgd::make_tma_map_bf16(&t.A.map, A, Kd, M, G, Kd, (uint64_t)M * Kd, 64, lsgd::kTcTileM);
      t.A.box_rows = lsgd::kTcTileM;
    }
    const int bn = lsgd::tc_tile_n(Kd);
    if (b_mn) {
      ok &= lsgd::make_tma_map_bf16(&t.B.map, B, N, Kd, G, N, (uint64_t)N * Kd, 64, 64);
      t.B.box_rows = 64;
    } else {
      ok &= lsgd::make_tma_map_bf16(&t.B.map, B, Kd, N, G, Kd, (uint64_t)N * Kd, 64, bn);
      t.B.box_rows = bn;
    }
    if (!ok) return fail(nullptr, LSGD_ECUDA, "TMA map encoding failed");
    t.A.mn_major = a_mn != 0;
    t.B.mn_major = b_mn != 0;
    t.C = C;
    t.c_rs = N;
    t.c_gs = (int64_t)M * N;
    t.c_bf16 = false;
    t.epi = lsgd::EPI_STORE;
    e = lsgd::launch_gemm_tc(t, s);
  } else {
    lsgd::GemmArgs g{};
    g.M = M;
    g.N = N;
    g.Kd = Kd;
    g.G = G;
    g.A = A;
    g.a_rs = a_mn ? 1 : Kd;
    g.a_cs = a_mn ? M : 1;
    g.a_gs = (int64_t)M * Kd;
    g.a_bf16 = true;
    g.B = B;  // B(k, n) = B[g](n, k)
    g.b_rs = b_mn ? N : 1;
    g.b_cs = b_mn ? 1 : Kd;
    g.b_gs = (int64_t)N * Kd;
    g.b_bf16 = true;
    g.C = C;
    g.c_rs = N;
    g.c_gs = (int64_t)M * N;
    g.c_bf16 = false;
    g.epi = lsgd::EPI_STORE;
    e = lsgd::launch_gemm_simt(g, s);
  }
  if (e != cudaSuccess) return fail_cuda(nullptr, e, "lsgd_grouped_gemm_bf16");
  return LSGD_OK;
}

lsgd_status lsgd_batchnorm_stats(const float* y, int64_t P, int C, int G, float* mean, float* rstd,
                                 void* stream) {
  if (!y || !mean || !rstd || P < 1 || C < 1 || C > 256 || G < 1 || G > 65535 ||
      (P + 1023) / 1024 > 65535)
    return fail(nullptr, LSGD_EINVAL, "lsgd_batchnorm_stats: bad arguments");
  cudaStream_t s = (cudaStream_t)stream;
  float* part = nullptr;
  const size_t bytes = lsgd::batchnorm_stats_scratch_floats(P, C, G) * sizeof(float);
  if (cudaMallocAsync((void**)&part, bytes, s) != cudaSuccess) {
    cudaGetLastError();
    return fail(nullptr, LSGD_ENOMEM, "lsgd_batchnorm_stats: scratch allocation failed");
  }
  cudaError_t e = lsgd::launch_batchnorm_stats(y, P, C, G, mean, rstd, part, s);
  cudaFreeAsync(part, s);
  if (e != cudaSuccess) return fail_cuda(nullptr, e, "lsgd_batchnorm_stats");
  return LSGD_OK;
}

lsgd_status lsgd_conv_wgrad_bf16(const uint16_t* x, const uint16_t* dy, float* dW, int G, int B,
                                 int Hout, int Wout, int Cin, int Cout, int stride, void* stream) {
  if (!x || !dy || !dW || G < 1 || G > 65535 || B < 1 ||
      !lsgd::conv_wgrad_tc_ok(Cin, Cout, stride, Hout * stride, Wout * stride, Hout, Wout) ||
      (int64_t)B * Hout * Wout > 0x7fffffffLL)
    return fail(nullptr, LSGD_EINVAL, "lsgd_conv_wgrad_bf16: bad arguments");
  if (((uintptr_t)x & 15) || ((uintptr_t)dy & 15))
    return fail(nullptr, LSGD_EINVAL, "lsgd_conv_wgrad_bf16: operands must be 16-byte aligned");
  if (!lsgd::tc_available()) return fail(nullptr, LSGD_EUNSUPPORTED, "tcgen05 not available");
  cudaStream_t s = (cudaStream_t)stream;
  float* part = nullptr;
  const size_t bytes =
      lsgd::conv_wgrad_scratch_floats(G, B, Hout, Wout, Cin, Cout, stride) * sizeof(float);
  if (cudaMallocAsync((void**)&part, bytes, s) != cudaSuccess) {
    cudaGetLastError();
    return fail(nullptr, LSGD_ENOMEM, "lsgd_conv_wgrad_bf16: scratch allocation failed");
  }
  cudaError_t e = lsgd::launch_conv_wgrad_bf16(x, dy, dW, (int64_t)Cout * 9 * Cin, G, B, Hout, Wout,
                                               Cin, Cout, stride, part, s);
  cudaFreeAsync(part, s);
  if (e != cudaSuccess) return fail_cuda(nullptr, e, "lsgd_conv_wgrad_bf16");
  return LSGD_OK;
}

lsgd_status lsgd_conv3x3_bf16(int mode, const uint16_t* in, const uint16_t* W, float* out, int G,
                              int B, int Hin, int Win, int Cin, int Cout, int stride,
                              void* stream) {
  if (!in || !W || !out || (mode != 0 && mode != 1) || G < 1 || G > 65535 || B < 1 || Hin < 1 ||
      Win < 1 || Cin < 1 || Cout < 1 || (stride != 1 && stride != 2))
    return fail(nullptr, LSGD_EINVAL, "lsgd_conv3x3_bf16: bad arguments");
  if (((uintptr_t)in & 15) || ((uintptr_t)W & 15))
    return fail(nullptr, LSGD_EINVAL, "lsgd_conv3x3_bf16: operands must be 16-byte aligned");
  if (!lsgd::tc_available()) return fail(nullptr, LSGD_EUNSUPPORTED, "tcgen05 not available");
  if (!lsgd::conv3x3_tc_route(mode, B, Hin, Win, Cin, Cout, stride))
    return fail(nullptr, LSGD_EUNSUPPORTED,
                "lsgd_conv3x3_bf16: shape not taken by the implicit-GEMM convolution kernel");
  cudaStream_t s = (cudaStream_t)stream;
  void* scratch = nullptr;
  const size_t bytes = lsgd::conv3x3_scratch_bytes(mode, G, B, Hin, Win, Cin, Cout, stride);
  if (bytes && cudaMallocAsync(&scratch, bytes, s) != cudaSuccess) {
    cudaGetLastError();
    return fail(nullptr, LSGD_ENOMEM, "lsgd_conv3x3_bf16: scratch allocation failed");
  }
  std::string err;
  const lsgd_status st = lsgd::conv3x3_bf16(mode, in, W, out, G, B, Hin, Win, Cin, Cout, stride,
                                            scratch, s, &err);
  if (scratch) cudaFreeAsync(scratch, s);
  if (st != LSGD_OK) return fail(nullptr, st, ("lsgd_conv3x3_bf16: " + err).c_str());
  return LSGD_OK;
}

lsgd_status lsgd_conv3x3_bn_bf16(const uint16_t* x, const uint16_t* W, float* y, float* mean,
                                 float* rstd, int G, int B, int Hin, int Win, int Cin, int Cout,
                                 int stride, void* stream) {
  if (!x || !W || !y || !mean || !rstd || G < 1 || G > 65535 || B < 1 || Hin < 1 || Win < 1 ||
      Cin < 1 || Cout < 1 || (stride != 1 && stride != 2))
    return fail(nullptr, LSGD_EINVAL, "lsgd_conv3x3_bn_bf16: bad arguments");
  if (((uintptr_t)x & 15) || ((uintptr_t)W & 15))
    return fail(nullptr, LSGD_EINVAL, "lsgd_conv3x3_bn_bf16: operands must be 16-byte aligned");
  if (!lsgd::tc_available()) return fail(nullptr, LSGD_EUNSUPPORTED, "tcgen05 not available");
  if (!lsgd::conv3x3_tc_route(0, B, Hin, Win, Cin, Cout, stride) || Cout > 64)
    return fail(nullptr, LSGD_EUNSUPPORTED,
                "lsgd_conv3x3_bn_bf16: shape not taken by the implicit-GEMM convolution kernel");
  cudaStream_t s = (cudaStream_t)stream;
  void* scratch = nullptr;
  const size_t bytes = lsgd::conv3x3_bn_scratch_bytes(G, B, Hin, Win, Cin, Cout, stride);
  if (cudaMallocAsync(&scratch, bytes, s) != cudaSuccess) {
    cudaGetLastError();
    return fail(nullptr, LSGD_ENOMEM, "lsgd_conv3x3_bn_bf16: scratch allocation failed");
  }
  std::string err;
  const lsgd_status st = lsgd::conv3x3_bn_bf16(x, W, y, mean, rstd, G, B, Hin, Win, Cin, Cout,
                                               stride, scratch, s, &err);
  cudaFreeAsync(scratch, s);
  if (st != LSGD_OK) return fail(nullptr, st, ("lsgd_conv3x3_bn_bf16: " + err).c_str());
  return LSGD_OK;
}

lsgd_status lsgd_sample_indices(int32_t* dst, uint64_t seed, int64_t step, int K, int B, int64_t N,
                                void* stream) {
  if (!dst || K < 1 || B < 1 || N < K) return fail(nullptr, LSGD_EINVAL, "lsgd_sample_indices: bad arguments");
  cudaError_t e =
      lsgd::launch_sample_indices(dst, seed, step, K, B, N, LSGD_SAMPLE_SHARDS, (cudaStream_t)stream);
  if (e != cudaSuccess) return fail_cuda(nullptr, e, "lsgd_sample_indices");
  return LSGD_OK;
}

}  // extern "C"
