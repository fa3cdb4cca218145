// Oracle driver and dense models -- TEST INFRASTRUCTURE ONLY (see oracle.h).
//
// Plain fp64 restatement of the method, one worker after another, one sample after another.  Each
// function names the passage of the paper it follows.  Nothing here is blocked, fused or reordered
// beyond what the cited definition states.
#include "oracle.h"

#include <cmath>
#include <cstdint>
#include <cstring>
#include <vector>

#include "philox.h"

namespace oracle {
// ResNet-20 pieces live in resnet.cpp.
int64_t resnet_num_params(const oracle_cfg* c);
void resnet_init(const oracle_cfg* c, uint64_t seed, double* w);
void resnet_wd_mask(const oracle_cfg* c, uint8_t* mask);
double resnet_loss_grad(const oracle_cfg* c, const double* w, const float* X, const int32_t* y,
                        const int32_t* idx, int B, double* grad);
double normal_from_philox(uint64_t seed, uint32_t tensor_id, uint32_t q);
double bf16_round(double x);
}  // namespace oracle

namespace oracle {

// bf16 storage of a value: the accelerated path holds fp32 values and stores GEMM operands as
// bf16 with round-to-nearest-even, so the oracle rounds fp64 -> fp32 -> bf16 the same way.
double bf16_round(double x) {
  float f = (float)x;
  uint32_t u;
  std::memcpy(&u, &f, 4);
  if ((u & 0x7f800000u) == 0x7f800000u) return x;  // inf / nan pass through
  const uint32_t lsb = (u >> 16) & 1u;
  u += 0x7fffu + lsb;
  u &= 0xffff0000u;
  std::memcpy(&f, &u, 4);
  return (double)f;
}

// A standard normal draw for element q of parameter tensor `tensor_id` (initialisation stream,
// counter word 3 = 1): Box-Muller on two Philox words mapped to the open interval (0, 1).
double normal_from_philox(uint64_t seed, uint32_t tensor_id, uint32_t q) {
  Philox4 ctr = {{q >> 2, tensor_id, 0u, 1u}};
  Philox4 r = philox4x32_10(ctr, (uint32_t)seed, (uint32_t)(seed >> 32));
  const int pair = (q >> 1) & 1;
  const double u1 = ((double)r.v[2 * pair] + 0.5) * (1.0 / 4294967296.0);
  const double u2 = ((double)r.v[2 * pair + 1] + 0.5) * (1.0 / 4294967296.0);
  const double radius = std::sqrt(-2.0 * std::log(u1));
  const double theta = 2.0 * M_PI * u2;
  return (q & 1) ? radius * std::sin(theta) : radius * std::cos(theta);
}

namespace {

int64_t dense_num_params(const oracle_cfg* c) {
  int64_t d = 0;
  for (int l = 0; l < c->n_layers; ++l) {
    d += (int64_t)c->widths[l] * c->widths[l + 1];
    if (c->has_bias) d += c->widths[l + 1];
  }
  return d;
}

// Eq. 2's local gradient (1/B) sum_{i in I} grad f_i(w) for a dense network: layers
// z_l = a_{l-1} W_l^T + b_l, a_l = relu(z_l) between layers, softmax cross-entropy on the last
// layer (kind DENSE) or f_i = 1/2 (a_i^T w - t_i)^2 (kind LSQ).  Returns the mean loss of the batch.
double dense_loss_grad(const oracle_cfg* c, const double* w, const float* X, const int32_t* y,
                       const float* t, const int32_t* idx, int B, double* grad) {
  const int L = c->n_layers;
  const bool q = c->bf16 != 0;
  auto rnd = [q](double v) { return q ? bf16_round(v) : v; };

  // Parameter views (canonical order: W_1, b_1, W_2, b_2, ...).
  std::vector<const double*> W(L), b(L);
  std::vector<double*> gW(L), gb(L);
  int64_t off = 0;
  for (int l = 0; l < L; ++l) {
    const int in = c->widths[l], out = c->widths[l + 1];
    W[l] = w + off;
    gW[l] = grad + off;
    off += (int64_t)in * out;
    if (c->has_bias) {
      b[l] = w + off;
      gb[l] = grad + off;
      off += out;
    } else {
      b[l] = nullptr;
      gb[l] = nullptr;
    }
  }

  // Forward.  a[l] holds the (stored) input of layer l+1; in bf16 mode that is the bf16 value.
  std::vector<std::vector<double>> a(L + 1);
  const int D = c->widths[0];
  a[0].resize((size_t)B * D);
  for (int j = 0; j < B; ++j)
    for (int i = 0; i < D; ++i) a[0][(size_t)j * D + i] = rnd((double)X[(size_t)idx[j] * D + i]);
  std::vector<double> logits;
  for (int l = 0; l < L; ++l) {
    const int in = c->widths[l], out = c->widths[l + 1];
    std::vector<double> Wq((size_t)in * out);
    for (size_t e = 0; e < Wq.size(); ++e) Wq[e] = rnd(W[l][e]);
    std::vector<double> z((size_t)B * out);
    for (int j = 0; j < B; ++j)
      for (int o = 0; o < out; ++o) {
        double acc = 0.0;
        for (int i = 0; i < in; ++i) acc += a[l][(size_t)j * in + i] * Wq[(size_t)o * in + i];
        if (b[l]) acc += b[l][o];
        z[(size_t)j * out + o] = acc;
      }
    if (l + 1 < L) {
      a[l + 1].resize(z.size());
      for (size_t e = 0; e < z.size(); ++e) a[l + 1][e] = rnd(z[e] > 0.0 ? z[e] : 0.0);
    } else {
      logits = z;
    }
  }

  // Loss and its gradient with respect to the last layer's output (already scaled by 1/B).
  const int C = c->widths[L];
  std::vector<double> dz((size_t)B * C);
  double loss = 0.0;
  for (int j = 0; j < B; ++j) {
    const double* zj = &logits[(size_t)j * C];
    if (c->kind == ORACLE_LSQ) {
      const double r = zj[0] - (double)t[idx[j]];
      loss += 0.5 * r * r;
      dz[j] = r / B;
    } else {
      double mx = zj[0];
      for (int k = 1; k < C; ++k) mx = zj[k] > mx ? zj[k] : mx;
      double se = 0.0;
      for (int k = 0; k < C; ++k) se += std::exp(zj[k] - mx);
      const double lse = mx + std::log(se);
      loss += lse - zj[y[idx[j]]];
      for (int k = 0; k < C; ++k) {
        const double p = std::exp(zj[k] - lse);
        dz[(size_t)j * C + k] = (p - (k == y[idx[j]] ? 1.0 : 0.0)) / B;
      }
    }
  }
  loss /= B;

  // Backward through the layers, last to first.
  for (int l = L - 1; l >= 0; --l) {
    const int in = c->widths[l], out = c->widths[l + 1];
    std::vector<double> dzq(dz.size());
    for (size_t e = 0; e < dz.size(); ++e) dzq[e] = rnd(dz[e]);
    for (int o = 0; o < out; ++o)
      for (int i = 0; i < in; ++i) {
        double acc = 0.0;
        for (int j = 0; j < B; ++j) acc += dzq[(size_t)j * out + o] * a[l][(size_t)j * in + i];
        gW[l][(size_t)o * in + i] = acc;
      }
    if (gb[l])
      for (int o = 0; o < out; ++o) {
        double acc = 0.0;
        for (int j = 0; j < B; ++j) acc += dzq[(size_t)j * out + o];
        gb[l][o] = acc;
      }
    if (l > 0) {
      std::vector<double> Wq((size_t)in * out);
      for (size_t e = 0; e < Wq.size(); ++e) Wq[e] = rnd(W[l][e]);
      std::vector<double> dprev((size_t)B * in);
      for (int j = 0; j < B; ++j)
        for (int i = 0; i < in; ++i) {
          double acc = 0.0;
          for (int o = 0; o < out; ++o) acc += dzq[(size_t)j * out + o] * Wq[(size_t)o * in + i];
          // relu'(z) taken from the stored activation: a > 0 exactly when z > 0.
          dprev[(size_t)j * in + i] = a[l][(size_t)j * in + i] > 0.0 ? acc : 0.0;
        }
      dz.swap(dprev);
    }
  }
  return loss;
}

void dense_init(const oracle_cfg* c, double* w) {
  int64_t off = 0;
  for (int l = 0; l < c->n_layers; ++l) {
    const int in = c->widths[l], out = c->widths[l + 1];
    const double sd = std::sqrt(2.0 / in);  // He et al. 2015, fan-in form
    for (int64_t e = 0; e < (int64_t)in * out; ++e)
      w[off + e] = (double)(float)(sd * normal_from_philox(c->seed, (uint32_t)l, (uint32_t)e));
    off += (int64_t)in * out;
    if (c->has_bias) {
      for (int o = 0; o < out; ++o) w[off + o] = 0.0;
      off += out;
    }
  }
}

}  // namespace
}  // namespace oracle

using namespace oracle;

extern "C" {

double oracle_bf16_round(double x) { return bf16_round(x); }

int64_t oracle_num_params(const oracle_cfg* c) {
  if (c->kind == ORACLE_RESNET20) return resnet_num_params(c);
  return dense_num_params(c);
}

// Weight decay applies to every parameter except the BatchNorm affine coefficients (Sec. A.4).
void oracle_weight_decay_mask(const oracle_cfg* c, uint8_t* mask) {
  if (c->kind == ORACLE_RESNET20) {
    resnet_wd_mask(c, mask);
    return;
  }
  const int64_t d = dense_num_params(c);
  for (int64_t i = 0; i < d; ++i) mask[i] = 1;
}

void oracle_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
  Philox4 p = {{ctr[0], ctr[1], ctr[2], ctr[3]}};
  Philox4 r = philox4x32_10(p, key[0], key[1]);
  for (int i = 0; i < 4; ++i) out[i] = r.v[i];
}

// Mini-batch I^k_s of worker k at local step s (Eq. 1 / Eq. 2: drawn uniformly, with replacement,
// from the worker's local data).  The data is split into K contiguous shards of floor(N/K) points;
// draw j uses word (j mod 4) of Philox(counter = (j div 4, s, k, 0), key = seed) and maps it to the
// shard by the high half of a 32x32-bit product.
int64_t oracle_epoch(const oracle_cfg* c, int64_t s) {
  return s * (int64_t)c->K * c->B / c->N;
}

// The reshuffling sampler's permutation of [0, N) for epoch e: a balanced Feistel network of four
// rounds (Luby and Rackoff) on the smallest even-bit domain 2^(2h) >= N, with round functions
// F_r(R) = word 0 of Philox4x32-10((R, e, r, 2), seed) masked to h bits, restricted to [0, N) by
// cycle walking (Black and Rogaway): apply the network until the value falls inside [0, N).  Each
// network is a bijection of the domain, so the walk from any i < N returns to [0, N) and the result
// is a bijection of [0, N).
int64_t oracle_permute(const oracle_cfg* c, int64_t e, int64_t i) {
  int h = 1;
  while ((int64_t)1 << (2 * h) < c->N) ++h;
  const uint64_t mask = ((uint64_t)1 << h) - 1;
  uint64_t x = (uint64_t)i;
  do {
    uint64_t L = x >> h, R = x & mask;
    for (uint32_t r = 0; r < 4; ++r) {
      Philox4 ctr = {{(uint32_t)R, (uint32_t)e, r, 2u}};
      const Philox4 f = philox4x32_10(ctr, (uint32_t)c->seed, (uint32_t)(c->seed >> 32));
      const uint64_t nR = L ^ ((uint64_t)f.v[0] & mask);
      L = R;
      R = nR;
    }
    x = (L << h) | R;
  } while (x >= (uint64_t)c->N);
  return (int64_t)x;
}

// I^k_s.  Shards: static contiguous shard of S = floor(N / K) points, B uniform draws with
// replacement.  Reshuffle: in epoch e the data is pi_e(0), ..., pi_e(N - 1), worker k's partition
// is positions [k S, (k + 1) S) of it, and the worker's t-th step of the epoch takes the next B
// positions of its partition, (t B + j) mod S.
void oracle_sample_indices(const oracle_cfg* c, int k, int64_t s, int32_t* out) {
  const uint64_t S = (uint64_t)(c->N / c->K);
  const uint64_t base = (uint64_t)k * S;
  if (c->sampling == ORACLE_SAMPLE_RESHUFFLE) {
    const int64_t e = oracle_epoch(c, s);
    const int64_t KB = (int64_t)c->K * c->B;
    const int64_t first = (e * c->N + KB - 1) / KB;  // first step of epoch e
    const int64_t t = s - first;
    for (int j = 0; j < c->B; ++j) {
      const uint64_t pos = ((uint64_t)t * c->B + j) % S;
      out[j] = (int32_t)oracle_permute(c, e, (int64_t)(base + pos));
    }
    return;
  }
  for (int j = 0; j < c->B; ++j) {
    Philox4 ctr = {{(uint32_t)(j >> 2), (uint32_t)s, (uint32_t)k, 0u}};
    Philox4 r = philox4x32_10(ctr, (uint32_t)c->seed, (uint32_t)(c->seed >> 32));
    const uint64_t word = r.v[j & 3];
    out[j] = (int32_t)(base + ((word * S) >> 32));
  }
}

// w_(0): He-normal weights (Sec. A.2 for convolutions; the dense models use the fan-in He rule),
// zero biases; or all zeros.
void oracle_init_params(const oracle_cfg* c, int init_kind, double* w) {
  const int64_t d = oracle_num_params(c);
  if (init_kind == ORACLE_INIT_ZERO) {
    for (int64_t i = 0; i < d; ++i) w[i] = 0.0;
    return;
  }
  if (c->kind == ORACLE_RESNET20)
    resnet_init(c, c->seed, w);
  else
    dense_init(c, w);
}

double oracle_loss_grad(const oracle_cfg* c, const double* w, const float* X, const int32_t* y,
                        const float* t, const int32_t* idx, int B, double* grad) {
  if (c->kind == ORACLE_RESNET20) return resnet_loss_grad(c, w, X, y, idx, B, grad);
  return dense_loss_grad(c, w, X, y, t, idx, B, grad);
}

// Local momentum SGD step on one worker (Sec. C.3.1: u = m u + grad, w = w - gamma u, kept per
// worker), with the Nesterov variant without dampening and plain L2 weight decay (Sec. A.4): g' = g + lambda w; u = m u + g'; step = g' + m u (Nesterov) or u; w -= gamma step.
// With the signSGD variant of Algorithm 4 the local step moves by lr sign(step), the step
// direction after weight decay and momentum (sign(0) = 0).
void oracle_sgd_update(const oracle_cfg* c, double lr, double* w, double* u, const double* g) {
  const int64_t d = oracle_num_params(c);
  std::vector<uint8_t> mask((size_t)d);
  oracle_weight_decay_mask(c, mask.data());
  for (int64_t i = 0; i < d; ++i) {
    const double gp = g[i] + (mask[i] ? c->weight_decay * w[i] : 0.0);
    double step;
    if (c->momentum == 0.0) {
      step = gp;
    } else {
      u[i] = c->momentum * u[i] + gp;
      step = c->nesterov ? gp + c->momentum * u[i] : u[i];
    }
    if (c->compress == ORACLE_COMPRESS_SIGN) step = (step > 0.0) - (step < 0.0);
    w[i] -= lr * step;
  }
}

// gamma(s): linear scaling by K and gradual warm-up (Sec. A.3: start at eta, add
// (eta_hat - eta) / (warmup_epochs * N / (K B)) per step until eta_hat), then multiply by `decay`
// once the run has used each milestone fraction of its samples (Sec. 4 / A.4: /10 at 50% and 75%).
double oracle_lr(const oracle_cfg* c, int64_t s) {
  const double eta = c->base_lr;
  const double eta_hat = c->scale_by_K ? eta * c->K : eta;
  double lr = eta_hat;
  if (c->warmup_epochs > 0.0 && eta_hat != eta) {
    const double steps_per_epoch = (double)c->N / ((double)c->K * c->B);
    const double inc = (eta_hat - eta) / (c->warmup_epochs * steps_per_epoch);
    const double v = eta + (double)s * inc;
    lr = v < eta_hat ? v : eta_hat;
  }
  for (int m = 0; m < c->n_milestones; ++m)
    if (s >= (int64_t)std::floor(c->milestones[m] * (double)c->T)) lr *= c->decay;
  return lr;
}

// Local-step warm-up: the round that starts in epoch e < P = h_warmup_epochs has length
//   linear:      1 + floor((H - 1) e / P)
//   exponential: min(H, 2^floor(e log2(H) / P))   (H = 8 over P = 3 epochs: 1, 2, 4, then 8)
//   constant:    1
// and H once e >= P.
int64_t oracle_round_length(const oracle_cfg* c, int64_t s0) {
  if (c->h_warmup == ORACLE_HWARM_NONE) return c->H;
  const double e = (double)oracle_epoch(c, s0), P = c->h_warmup_epochs;
  if (e >= P) return c->H;
  switch (c->h_warmup) {
    case ORACLE_HWARM_LINEAR:
      return 1 + (int64_t)std::floor((double)(c->H - 1) * e / P);
    case ORACLE_HWARM_EXPONENTIAL: {
      const double x = std::floor(e * std::log2((double)c->H) / P);
      const double len = std::pow(2.0, x);
      return len < (double)c->H ? (int64_t)len : c->H;
    }
    default:
      return 1;
  }
}

// Whether the models are averaged after local step s (0-based): post-local SGD (Sec. 3) uses
// H_(t) = 1 before the switch step t' and H after it; the last step of the run always ends a round
// so the returned model is the average.
int oracle_is_round_end(const oracle_cfg* c, int64_t s) {
  if (s == c->T - 1) return 1;
  if (c->t_switch >= 0 && s < c->t_switch) return 1;
  const int64_t start = c->t_switch > 0 ? c->t_switch : 0;
  if (c->h_warmup == ORACLE_HWARM_NONE) return ((s + 1 - start) % c->H) == 0;
  // rounds of varying length, walked from the first one
  int64_t r0 = start;
  for (;;) {
    const int64_t len = oracle_round_length(c, r0);
    if (s < r0 + len) return s == r0 + len - 1;
    r0 += len;
  }
}

// Which average ends local step s.  Without hierarchy: the global average at every round end.
// Hierarchical local SGD (Sec. D, the equations of the hierarchical scheme): the r-th round end
// after the switch averages within each block of hier_block workers, and every hier_rounds-th
// round end (r a multiple of H^b) averages all K workers; the mini-batch phase (s < t') and the
// last step of the run use the global average.
int oracle_sync_kind(const oracle_cfg* c, int64_t s) {
  if (!oracle_is_round_end(c, s)) return ORACLE_SYNC_NONE;
  if (c->hier_block <= 0 || s == c->T - 1) return ORACLE_SYNC_GLOBAL;
  if (c->t_switch >= 0 && s < c->t_switch) return ORACLE_SYNC_GLOBAL;
  const int64_t start = c->t_switch > 0 ? c->t_switch : 0;
  const int64_t r = (s + 1 - start) / c->H;
  return (r % c->hier_rounds == 0) ? ORACLE_SYNC_GLOBAL : ORACLE_SYNC_BLOCK;
}

// Block average: w^k := (1/K') sum over the K' workers of k's block (Sec. D).
void oracle_block_average(int K, int block, int64_t d, double* W) {
  for (int b0 = 0; b0 < K; b0 += block) oracle_average(block, d, W + (int64_t)b0 * d);
}

// Eq. 2, right part: w^k := (1/K) sum_k w^k for every worker k.
void oracle_average(int K, int64_t d, double* W) {
  for (int64_t i = 0; i < d; ++i) {
    double acc = 0.0;
    for (int k = 0; k < K; ++k) acc += W[(int64_t)k * d + i];
    const double mean = acc / K;
    for (int k = 0; k < K; ++k) W[(int64_t)k * d + i] = mean;
  }
}

// Local / post-local SGD (Eq. 2; Algorithms 1 and 2) from global step s0 for n_steps steps.
// W and U hold the K workers' models and momentum buffers, worker-major, and are updated in place.
namespace {

// The synchronisation that ends a round, for the round-start model wref shared by all workers:
//  * plain (Eq. 2): w^k := wref := (1/K) sum_k w^k;
//  * global momentum (Sec. C.3.1): ug := m_g ug + (wref - mean_k w^k) / lr; wref -= lr ug;
//  * signSGD compression (Algorithm 4): Delta^k = wref - w^k, s^k = sign(Delta^k),
//    p^k = ||Delta^k||_1 / d; wref -= (1/K) sum_k s^k p^k;
//  * EF-signSGD (Algorithm 5): Delta^k = wref - w^k + e^k, s^k, p^k as above,
//    e^k := Delta^k - s^k p^k (the residual the compression dropped), wref -= (1/K) sum_k s^k p^k;
// and every worker restarts from wref.
void global_sync(const oracle_cfg* c, int64_t d, double lr, double* W, double* wref, double* E,
                 double* ug) {
  const int K = c->K;
  if (c->compress == ORACLE_COMPRESS_NONE) {
    oracle_average(K, d, W);
    if (c->global_momentum > 0.0) {
      for (int64_t i = 0; i < d; ++i) {
        ug[i] = c->global_momentum * ug[i] + (wref[i] - W[i]) / lr;
        wref[i] -= lr * ug[i];
      }
      for (int k = 0; k < K; ++k)
        for (int64_t i = 0; i < d; ++i) W[(int64_t)k * d + i] = wref[i];
    } else {
      for (int64_t i = 0; i < d; ++i) wref[i] = W[i];
    }
    return;
  }
  std::vector<double> delta((size_t)K * d), p((size_t)K);
  for (int k = 0; k < K; ++k) {
    double l1 = 0.0;
    for (int64_t i = 0; i < d; ++i) {
      double v = wref[i] - W[(int64_t)k * d + i];
      if (c->compress == ORACLE_COMPRESS_EF_SIGN) v += E[(int64_t)k * d + i];
      delta[(size_t)k * d + i] = v;
      l1 += std::fabs(v);
    }
    p[k] = l1 / (double)d;
  }
  for (int64_t i = 0; i < d; ++i) {
    double acc = 0.0;
    for (int k = 0; k < K; ++k) {
      const double v = delta[(size_t)k * d + i];
      const double sp = (double)((v > 0.0) - (v < 0.0)) * p[k];
      acc += sp;
      if (c->compress == ORACLE_COMPRESS_EF_SIGN) E[(int64_t)k * d + i] = v - sp;
    }
    wref[i] -= acc / K;
  }
  for (int k = 0; k < K; ++k)
    for (int64_t i = 0; i < d; ++i) W[(int64_t)k * d + i] = wref[i];
}

}  // namespace

void oracle_run_ext(const oracle_cfg* c, const float* X, const int32_t* y, const float* t,
                    double* W, double* U, double* Wref, double* E, double* Ug, int64_t s0,
                    int64_t n_steps, double* losses, int64_t* n_global, int64_t* n_block) {
  const int64_t d = oracle_num_params(c);
  std::vector<int32_t> idx((size_t)c->B);
  std::vector<double> g((size_t)d);
  std::vector<double> wref_own, e_own, ug_own;
  if (!Wref) {
    wref_own.assign(W, W + d);
    Wref = wref_own.data();
  }
  if (!E) {
    e_own.assign((size_t)c->K * d, 0.0);
    E = e_own.data();
  }
  if (!Ug) {
    ug_own.assign((size_t)d, 0.0);
    Ug = ug_own.data();
  }
  int64_t syncs = 0, blocks = 0;
  for (int64_t s = s0; s < s0 + n_steps; ++s) {
    const double lr = oracle_lr(c, s);
    for (int k = 0; k < c->K; ++k) {
      oracle_sample_indices(c, k, s, idx.data());
      const double l = oracle_loss_grad(c, W + (int64_t)k * d, X, y, t, idx.data(), c->B, g.data());
      oracle_sgd_update(c, lr, W + (int64_t)k * d, U + (int64_t)k * d, g.data());
      if (losses) losses[(s - s0) * c->K + k] = l;
    }
    const int kind = oracle_sync_kind(c, s);
    if (kind == ORACLE_SYNC_GLOBAL) {
      global_sync(c, d, lr, W, Wref, E, Ug);
      ++syncs;
    } else if (kind == ORACLE_SYNC_BLOCK) {
      oracle_block_average(c->K, c->hier_block, d, W);
      ++blocks;
    }
  }
  if (n_global) *n_global = syncs;
  if (n_block) *n_block = blocks;
}

void oracle_run_counted(const oracle_cfg* c, const float* X, const int32_t* y, const float* t,
                        double* W, double* U, int64_t s0, int64_t n_steps, double* losses,
                        int64_t* n_global, int64_t* n_block) {
  oracle_run_ext(c, X, y, t, W, U, nullptr, nullptr, nullptr, s0, n_steps, losses, n_global,
                 n_block);
}

void oracle_run(const oracle_cfg* c, const float* X, const int32_t* y, const float* t, double* W,
                double* U, int64_t s0, int64_t n_steps, double* losses, int64_t* n_syncs) {
  oracle_run_counted(c, X, y, t, W, U, s0, n_steps, losses, n_syncs, nullptr);
}

// Mini-batch SGD (Eq. 1) on a single model: each step averages the K workers' local mini-batch
// gradients, (1/K) sum_k (1/B) sum_{i in I^k} grad f_i(w), and applies one momentum-SGD step with a
// single (global) momentum buffer.  Written independently of oracle_run so the paper's special
// cases (H = 1, K = 1) can be checked against it.
void oracle_run_minibatch(const oracle_cfg* c, const float* X, const int32_t* y, const float* t,
                          double* w, double* u, int64_t s0, int64_t n_steps, double* losses) {
  const int64_t d = oracle_num_params(c);
  std::vector<int32_t> idx((size_t)c->B);
  std::vector<double> gk((size_t)d), g((size_t)d);
  for (int64_t s = s0; s < s0 + n_steps; ++s) {
    for (int64_t i = 0; i < d; ++i) g[i] = 0.0;
    double loss = 0.0;
    for (int k = 0; k < c->K; ++k) {
      oracle_sample_indices(c, k, s, idx.data());
      loss += oracle_loss_grad(c, w, X, y, t, idx.data(), c->B, gk.data());
      for (int64_t i = 0; i < d; ++i) g[i] += gk[i];
    }
    for (int64_t i = 0; i < d; ++i) g[i] /= c->K;
    oracle_sgd_update(c, oracle_lr(c, s), w, u, g.data());
    if (losses) losses[s - s0] = loss / c->K;
  }
}

// Mean training loss of model w over the first n data points (no gradient).
double oracle_eval_loss(const oracle_cfg* c, const double* w, const float* X, const int32_t* y,
                        const float* t, int64_t n) {
  const int64_t d = oracle_num_params(c);
  std::vector<double> g((size_t)d);
  const int chunk = 256;
  double total = 0.0;
  std::vector<int32_t> idx(chunk);
  for (int64_t start = 0; start < n; start += chunk) {
    const int b = (int)((n - start) < chunk ? (n - start) : chunk);
    for (int j = 0; j < b; ++j) idx[j] = (int32_t)(start + j);
    total += oracle_loss_grad(c, w, X, y, t, idx.data(), b, g.data()) * b;
  }
  return total / (double)n;
}

}  // extern "C"
