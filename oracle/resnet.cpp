// ResNet-20 (CIFAR form) for the oracle -- TEST INFRASTRUCTURE ONLY (see oracle.h).
//
// The network of He et al. 2016 used by the paper (Sec. 4 and A.2; 0.27 M parameters, Table
// "scaling ratio"): a 3x3 stem convolution, three stages of `res_blocks` basic blocks with
// base_ch, 2 base_ch, 4 base_ch channels (stride 2 at the first block of stages 2 and 3), the
// parameter-free "option A" shortcut (spatial subsampling by 2 plus zero channels appended after
// the input channels), BatchNorm with the worker's own batch statistics (Sec. A.4), global average
// pooling and a fully connected classifier.  Images are stored HWC (channel fastest); activations
// NHWC; convolution weights [Cout][3][3][Cin].  fp64 throughout; in bf16 mode the convolution
// operands (input activation, weight, output gradient) are rounded to bf16 where the accelerated
// path stores them in bf16 (the stored block outputs, inner activations and the image).
#include <cmath>
#include <cstdint>
#include <vector>

#include "oracle.h"

namespace oracle {
double normal_from_philox(uint64_t seed, uint32_t tensor_id, uint32_t q);
double bf16_round(double x);

namespace {

const double kBnEps = 1e-5;

struct ConvSpec {
  int cin, cout, stride;
  int64_t w_off, g_off, b_off;  // conv weight, BN gamma, BN beta offsets
};

struct Net {
  int H0, W0, C0, base, blocks, classes;
  ConvSpec stem;
  std::vector<ConvSpec> convs;  // 2 per block, block-major
  int64_t fc_w, fc_b, total;
};

Net make_net(const oracle_cfg* c) {
  Net n;
  n.H0 = c->in_h;
  n.W0 = c->in_w;
  n.C0 = c->in_c;
  n.base = c->base_ch;
  n.blocks = c->res_blocks;
  n.classes = c->n_classes;
  int64_t off = 0;
  auto add_conv = [&off](int cin, int cout, int stride) {
    ConvSpec s;
    s.cin = cin;
    s.cout = cout;
    s.stride = stride;
    s.w_off = off;
    off += (int64_t)cout * 9 * cin;
    s.g_off = off;
    off += cout;
    s.b_off = off;
    off += cout;
    return s;
  };
  n.stem = add_conv(n.C0, n.base, 1);
  int ch = n.base;
  for (int st = 0; st < 3; ++st) {
    const int cout = n.base << st;
    for (int b = 0; b < n.blocks; ++b) {
      const int stride = (st > 0 && b == 0) ? 2 : 1;
      n.convs.push_back(add_conv(ch, cout, stride));
      n.convs.push_back(add_conv(cout, cout, 1));
      ch = cout;
    }
  }
  n.fc_w = off;
  off += (int64_t)n.classes * ch;
  n.fc_b = off;
  off += n.classes;
  n.total = off;
  return n;
}

// Activation tensor [B][H][W][C].
struct Act {
  int B = 0, H = 0, W = 0, C = 0;
  std::vector<double> v;
  void init(int b, int h, int w, int c) {
    B = b;
    H = h;
    W = w;
    C = c;
    v.assign((size_t)b * h * w * c, 0.0);
  }
  double& at(int b, int h, int w, int c) { return v[(((size_t)b * H + h) * W + w) * C + c]; }
  double at(int b, int h, int w, int c) const { return v[(((size_t)b * H + h) * W + w) * C + c]; }
};

// 3x3 convolution, zero padding 1: out[b][oh][ow][co] = sum in[b][oh*s+kh-1][ow*s+kw-1][ci] w[co][kh][kw][ci].
void conv_fwd(const Act& in, const double* w, const ConvSpec& cs, Act& out) {
  const int Ho = (in.H - 1) / cs.stride + 1, Wo = (in.W - 1) / cs.stride + 1;
  out.init(in.B, Ho, Wo, cs.cout);
  for (int b = 0; b < in.B; ++b)
    for (int oh = 0; oh < Ho; ++oh)
      for (int ow = 0; ow < Wo; ++ow)
        for (int co = 0; co < cs.cout; ++co) {
          double acc = 0.0;
          for (int kh = 0; kh < 3; ++kh) {
            const int ih = oh * cs.stride + kh - 1;
            if (ih < 0 || ih >= in.H) continue;
            for (int kw = 0; kw < 3; ++kw) {
              const int iw = ow * cs.stride + kw - 1;
              if (iw < 0 || iw >= in.W) continue;
              for (int ci = 0; ci < cs.cin; ++ci)
                acc += in.at(b, ih, iw, ci) * w[(((size_t)co * 3 + kh) * 3 + kw) * cs.cin + ci];
            }
          }
          out.at(b, oh, ow, co) = acc;
        }
}

// Gradients of conv_fwd: dW[co][kh][kw][ci] = sum dy * in, din = sum dy * w (transposed conv).
void conv_bwd(const Act& in, const double* w, const ConvSpec& cs, const Act& dy, double* dW,
              Act* din) {
  for (int64_t e = 0; e < (int64_t)cs.cout * 9 * cs.cin; ++e) dW[e] = 0.0;
  if (din) din->init(in.B, in.H, in.W, in.C);
  for (int b = 0; b < dy.B; ++b)
    for (int oh = 0; oh < dy.H; ++oh)
      for (int ow = 0; ow < dy.W; ++ow)
        for (int co = 0; co < cs.cout; ++co) {
          const double g = dy.at(b, oh, ow, co);
          for (int kh = 0; kh < 3; ++kh) {
            const int ih = oh * cs.stride + kh - 1;
            if (ih < 0 || ih >= in.H) continue;
            for (int kw = 0; kw < 3; ++kw) {
              const int iw = ow * cs.stride + kw - 1;
              if (iw < 0 || iw >= in.W) continue;
              for (int ci = 0; ci < cs.cin; ++ci) {
                const size_t wi = (((size_t)co * 3 + kh) * 3 + kw) * cs.cin + ci;
                dW[wi] += g * in.at(b, ih, iw, ci);
                if (din) din->at(b, ih, iw, ci) += g * w[wi];
              }
            }
          }
        }
}

// BatchNorm with batch statistics over (B, H, W) per channel, biased variance (Ioffe & Szegedy).
struct BnCache {
  std::vector<double> mean, rstd;
  Act xhat;
};

void bn_fwd(const Act& y, const double* gamma, const double* beta, Act& out, BnCache& cache) {
  const int C = y.C;
  const size_t M = (size_t)y.B * y.H * y.W;
  cache.mean.assign(C, 0.0);
  cache.rstd.assign(C, 0.0);
  std::vector<double> var(C, 0.0);
  for (size_t p = 0; p < M; ++p)
    for (int ch = 0; ch < C; ++ch) cache.mean[ch] += y.v[p * C + ch];
  for (int ch = 0; ch < C; ++ch) cache.mean[ch] /= (double)M;
  for (size_t p = 0; p < M; ++p)
    for (int ch = 0; ch < C; ++ch) {
      const double dlt = y.v[p * C + ch] - cache.mean[ch];
      var[ch] += dlt * dlt;
    }
  for (int ch = 0; ch < C; ++ch) cache.rstd[ch] = 1.0 / std::sqrt(var[ch] / (double)M + kBnEps);
  cache.xhat.init(y.B, y.H, y.W, C);
  out.init(y.B, y.H, y.W, C);
  for (size_t p = 0; p < M; ++p)
    for (int ch = 0; ch < C; ++ch) {
      const double xh = (y.v[p * C + ch] - cache.mean[ch]) * cache.rstd[ch];
      cache.xhat.v[p * C + ch] = xh;
      out.v[p * C + ch] = gamma[ch] * xh + beta[ch];
    }
}

// dy = (gamma * rstd) (dz - mean(dz) - xhat mean(dz xhat)); dgamma = sum dz xhat; dbeta = sum dz.
void bn_bwd(const Act& dz, const double* gamma, const BnCache& cache, Act& dy, double* dgamma,
            double* dbeta) {
  const int C = dz.C;
  const size_t M = (size_t)dz.B * dz.H * dz.W;
  std::vector<double> sdz(C, 0.0), sdzx(C, 0.0);
  for (size_t p = 0; p < M; ++p)
    for (int ch = 0; ch < C; ++ch) {
      sdz[ch] += dz.v[p * C + ch];
      sdzx[ch] += dz.v[p * C + ch] * cache.xhat.v[p * C + ch];
    }
  dy.init(dz.B, dz.H, dz.W, C);
  for (int ch = 0; ch < C; ++ch) {
    dgamma[ch] = sdzx[ch];
    dbeta[ch] = sdz[ch];
  }
  for (size_t p = 0; p < M; ++p)
    for (int ch = 0; ch < C; ++ch) {
      const double mdz = sdz[ch] / (double)M, mdzx = sdzx[ch] / (double)M;
      dy.v[p * C + ch] =
          gamma[ch] * cache.rstd[ch] * (dz.v[p * C + ch] - mdz - cache.xhat.v[p * C + ch] * mdzx);
    }
}

// Option-A shortcut: x[:, ::s, ::s, :] with zero channels appended up to cout.
void shortcut_fwd(const Act& x, int stride, int cout, Act& out) {
  const int Ho = (x.H - 1) / stride + 1, Wo = (x.W - 1) / stride + 1;
  out.init(x.B, Ho, Wo, cout);
  for (int b = 0; b < x.B; ++b)
    for (int h = 0; h < Ho; ++h)
      for (int w = 0; w < Wo; ++w)
        for (int ch = 0; ch < x.C; ++ch) out.at(b, h, w, ch) = x.at(b, h * stride, w * stride, ch);
}

void shortcut_bwd(const Act& dout, int stride, Act& dx) {
  for (int b = 0; b < dout.B; ++b)
    for (int h = 0; h < dout.H; ++h)
      for (int w = 0; w < dout.W; ++w)
        for (int ch = 0; ch < dx.C; ++ch) dx.at(b, h * stride, w * stride, ch) += dout.at(b, h, w, ch);
}

struct ConvCache {
  Act in;  // the (stored) convolution input
  Act y;   // convolution output
  BnCache bn;
  Act act;  // stored post-activation output of this conv's BN (+ residual) + ReLU
};

}  // namespace

int64_t resnet_num_params(const oracle_cfg* c) { return make_net(c).total; }

void resnet_wd_mask(const oracle_cfg* c, uint8_t* mask) {
  Net n = make_net(c);
  for (int64_t i = 0; i < n.total; ++i) mask[i] = 1;
  auto clear_bn = [&](const ConvSpec& s) {
    for (int ch = 0; ch < s.cout; ++ch) {
      mask[s.g_off + ch] = 0;
      mask[s.b_off + ch] = 0;
    }
  };
  clear_bn(n.stem);
  for (const ConvSpec& s : n.convs) clear_bn(s);
}

// Sec. A.2: He initialisation for convolutions (fan-in = 9 Cin), N(0, 0.01^2) for the fully
// connected layer, zero biases; BatchNorm gamma = 1, beta = 0.
void resnet_init(const oracle_cfg* c, uint64_t seed, double* w) {
  Net n = make_net(c);
  uint32_t tensor = 0;
  auto init_conv = [&](const ConvSpec& s) {
    const double sd = std::sqrt(2.0 / (9.0 * s.cin));
    for (int64_t e = 0; e < (int64_t)s.cout * 9 * s.cin; ++e)
      w[s.w_off + e] = (double)(float)(sd * normal_from_philox(seed, tensor, (uint32_t)e));
    tensor++;
    for (int ch = 0; ch < s.cout; ++ch) {
      w[s.g_off + ch] = 1.0;
      w[s.b_off + ch] = 0.0;
    }
  };
  init_conv(n.stem);
  for (const ConvSpec& s : n.convs) init_conv(s);
  const int F = n.base * 4;
  for (int64_t e = 0; e < (int64_t)n.classes * F; ++e)
    w[n.fc_w + e] = (double)(float)(0.01 * normal_from_philox(seed, tensor, (uint32_t)e));
  for (int k = 0; k < n.classes; ++k) w[n.fc_b + k] = 0.0;
}

double resnet_loss_grad(const oracle_cfg* c, const double* w, const float* X, const int32_t* y,
                        const int32_t* idx, int B, double* grad) {
  const Net n = make_net(c);
  const bool q = c->bf16 != 0;
  auto rnd = [q](double v) { return q ? bf16_round(v) : v; };
  auto round_act = [&](Act& a) {
    if (q)
      for (double& v : a.v) v = bf16_round(v);
  };
  auto rounded_weights = [&](const ConvSpec& s) {
    std::vector<double> wq((size_t)s.cout * 9 * s.cin);
    for (size_t e = 0; e < wq.size(); ++e) wq[e] = rnd(w[s.w_off + e]);
    return wq;
  };
  for (int64_t i = 0; i < n.total; ++i) grad[i] = 0.0;

  // ---- forward ----
  Act x0;
  x0.init(B, n.H0, n.W0, n.C0);
  for (int b = 0; b < B; ++b)
    for (size_t e = 0; e < (size_t)n.H0 * n.W0 * n.C0; ++e)
      x0.v[(size_t)b * n.H0 * n.W0 * n.C0 + e] = (double)X[(size_t)idx[b] * n.H0 * n.W0 * n.C0 + e];
  round_act(x0);

  const size_t n_convs = n.convs.size();
  ConvCache stem;
  std::vector<ConvCache> cc(n_convs);
  std::vector<Act> sc(n_convs / 2);  // shortcut values per block

  stem.in = x0;
  {
    std::vector<double> wq = rounded_weights(n.stem);
    conv_fwd(stem.in, wq.data(), n.stem, stem.y);
    Act z;
    bn_fwd(stem.y, w + n.stem.g_off, w + n.stem.b_off, z, stem.bn);
    stem.act = z;
    for (double& v : stem.act.v) v = v > 0.0 ? v : 0.0;
    round_act(stem.act);
  }
  const Act* cur = &stem.act;
  for (size_t blk = 0; blk < n_convs / 2; ++blk) {
    ConvCache& A = cc[2 * blk];
    ConvCache& Bc = cc[2 * blk + 1];
    const ConvSpec& sa = n.convs[2 * blk];
    const ConvSpec& sb = n.convs[2 * blk + 1];
    A.in = *cur;
    std::vector<double> wa = rounded_weights(sa);
    conv_fwd(A.in, wa.data(), sa, A.y);
    Act za;
    bn_fwd(A.y, w + sa.g_off, w + sa.b_off, za, A.bn);
    A.act = za;
    for (double& v : A.act.v) v = v > 0.0 ? v : 0.0;
    round_act(A.act);
    Bc.in = A.act;
    std::vector<double> wb = rounded_weights(sb);
    conv_fwd(Bc.in, wb.data(), sb, Bc.y);
    Act zb;
    bn_fwd(Bc.y, w + sb.g_off, w + sb.b_off, zb, Bc.bn);
    shortcut_fwd(A.in, sa.stride, sa.cout, sc[blk]);
    Bc.act = zb;
    for (size_t e = 0; e < Bc.act.v.size(); ++e) {
      const double v = zb.v[e] + sc[blk].v[e];
      Bc.act.v[e] = v > 0.0 ? v : 0.0;
    }
    round_act(Bc.act);
    cur = &Bc.act;
  }

  // Global average pooling and the classifier (fp64; not a bf16 operand).
  const Act& last = *cur;
  const int F = last.C, HW = last.H * last.W, C = n.classes;
  std::vector<double> feat((size_t)B * F, 0.0);
  for (int b = 0; b < B; ++b)
    for (int p = 0; p < HW; ++p)
      for (int f = 0; f < F; ++f) feat[(size_t)b * F + f] += last.v[((size_t)b * HW + p) * F + f];
  for (double& v : feat) v /= (double)HW;
  std::vector<double> logits((size_t)B * C);
  for (int b = 0; b < B; ++b)
    for (int k = 0; k < C; ++k) {
      double acc = w[n.fc_b + k];
      for (int f = 0; f < F; ++f) acc += feat[(size_t)b * F + f] * w[n.fc_w + (size_t)k * F + f];
      logits[(size_t)b * C + k] = acc;
    }

  // ---- loss ----
  std::vector<double> dlog((size_t)B * C);
  double loss = 0.0;
  for (int b = 0; b < B; ++b) {
    const double* z = &logits[(size_t)b * C];
    double mx = z[0];
    for (int k = 1; k < C; ++k) mx = z[k] > mx ? z[k] : mx;
    double se = 0.0;
    for (int k = 0; k < C; ++k) se += std::exp(z[k] - mx);
    const double lse = mx + std::log(se);
    loss += lse - z[y[idx[b]]];
    for (int k = 0; k < C; ++k)
      dlog[(size_t)b * C + k] = (std::exp(z[k] - lse) - (k == y[idx[b]] ? 1.0 : 0.0)) / B;
  }
  loss /= B;

  // ---- backward ----
  for (int k = 0; k < C; ++k)
    for (int b = 0; b < B; ++b) grad[n.fc_b + k] += dlog[(size_t)b * C + k];
  for (int k = 0; k < C; ++k)
    for (int f = 0; f < F; ++f) {
      double acc = 0.0;
      for (int b = 0; b < B; ++b) acc += dlog[(size_t)b * C + k] * feat[(size_t)b * F + f];
      grad[n.fc_w + (size_t)k * F + f] = acc;
    }
  Act dcur;  // gradient w.r.t. the current stored activation
  dcur.init(B, last.H, last.W, F);
  for (int b = 0; b < B; ++b)
    for (int f = 0; f < F; ++f) {
      double acc = 0.0;
      for (int k = 0; k < C; ++k) acc += dlog[(size_t)b * C + k] * w[n.fc_w + (size_t)k * F + f];
      for (int p = 0; p < HW; ++p) dcur.v[((size_t)b * HW + p) * F + f] = acc / (double)HW;
    }

  auto relu_mask = [](Act& d, const Act& act) {
    for (size_t e = 0; e < d.v.size(); ++e)
      if (!(act.v[e] > 0.0)) d.v[e] = 0.0;
  };

  for (size_t blk = n_convs / 2; blk-- > 0;) {
    ConvCache& A = cc[2 * blk];
    ConvCache& Bc = cc[2 * blk + 1];
    const ConvSpec& sa = n.convs[2 * blk];
    const ConvSpec& sb = n.convs[2 * blk + 1];
    relu_mask(dcur, Bc.act);  // through the block's output ReLU
    Act dyb;
    bn_bwd(dcur, w + sb.g_off, Bc.bn, dyb, grad + sb.g_off, grad + sb.b_off);
    round_act(dyb);
    std::vector<double> wb = rounded_weights(sb);
    Act dh;
    conv_bwd(Bc.in, wb.data(), sb, dyb, grad + sb.w_off, &dh);
    relu_mask(dh, A.act);
    Act dya;
    bn_bwd(dh, w + sa.g_off, A.bn, dya, grad + sa.g_off, grad + sa.b_off);
    round_act(dya);
    std::vector<double> wa = rounded_weights(sa);
    Act dx;
    conv_bwd(A.in, wa.data(), sa, dya, grad + sa.w_off, &dx);
    shortcut_bwd(dcur, sa.stride, dx);  // residual path (the first A.in.C channels)
    dcur = dx;
  }
  relu_mask(dcur, stem.act);
  Act dys;
  bn_bwd(dcur, w + n.stem.g_off, stem.bn, dys, grad + n.stem.g_off, grad + n.stem.b_off);
  round_act(dys);
  std::vector<double> ws = rounded_weights(n.stem);
  conv_bwd(stem.in, ws.data(), n.stem, dys, grad + n.stem.w_off, nullptr);
  return loss;
}

}  // namespace oracle
