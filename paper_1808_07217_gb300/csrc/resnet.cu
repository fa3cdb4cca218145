// ResNet-20 on the CUDA path, K replicas per launch.
//
// The CIFAR network of He et al. 2016 used by the paper (Sec. 4 and A.2: 0.27 M parameters): a 3x3
// stem convolution, three stages of basic blocks (base, 2 base, 4 base channels; stride 2 at the
// first block of stages 2 and 3), option-A shortcuts (stride-2 subsampling, zero channels appended
// after the input channels), BatchNorm with each worker's own batch statistics (Sec. A.4), global
// average pooling and a fully connected classifier.  Activations are NHWC, replica-major
// ([K][B][H][W][C]); convolution weights [Cout][3][3][Cin].  In BF16 mode the convolution operands
// (image, stored activations, weights, output gradients) are bf16; accumulation, BatchNorm,
// pooling, the classifier and the update are fp32.
//
// Reductions over the pixels of a replica (BatchNorm statistics, their backward sums, weight
// gradients) run in two deterministic passes: per-chunk partial results into a scratch buffer,
// then a fixed-order combination.
//
// Every kernel here starts with the programmatic grid-dependency wait and is launched with
// programmatic dependent launch, so the next kernel's launch and prologue overlap this one's tail.
#include <algorithm>
#include <cmath>
#include <cstdlib>
#include <string>
#include <vector>

#include "common.cuh"
#include "lsgd_internal.h"
#include "resnet.h"

namespace lsgd {

namespace {

constexpr float kBnEps = 1e-5f;
constexpr int kStatChunk = 1024;   // pixels per BatchNorm reduction chunk (lsgd_batchnorm_stats)
constexpr int kRnChunk = 256;      // the smallest chunk inside the ResNet step (scratch sizing)
// Pixels per reduction chunk inside the ResNet step: 1024 on large tensors, 256 on the small
// later stages so that they still spread over many CTAs.
int rn_chunk(int64_t P) { return P >= 65536 ? 1024 : kRnChunk; }
constexpr int kWgradChunk = 2048;  // pixels per weight-gradient chunk
constexpr int kWgradTile = 16;     // pixels staged per weight-gradient iteration
constexpr int kMaxJ16 = 36;        // (9 Cin) / 16 accumulators per thread, Cin <= 64

struct ConvL {
  int cin, cout, stride, hin, win, hout, wout;
  int64_t w_off, g_off, b_off;  // padded per-replica offsets
  int64_t cw, cg, cb;           // canonical offsets
};

int64_t rup(int64_t v, int64_t m) { return (v + m - 1) / m * m; }

int grid_cap(int64_t items, int threads) {
  int64_t b = (items + threads - 1) / threads;
  return (int)std::max<int64_t>(1, std::min<int64_t>(b, (int64_t)kNumSMs * 16));
}

// ------------------------------------------------------------------------------------------
// Direct 3x3 convolution, zero padding 1: y[g][b][oh][ow][co] = sum_{kh,kw,ci}
// in[g][b][oh s + kh - 1][ow s + kw - 1][ci] w[g][co][kh][kw][ci].  One thread per output pixel
// and 16 output channels; the 16 channels' weights sit in shared memory.
template <typename TA>
__global__ void __launch_bounds__(128) conv_fwd_kernel(const TA* __restrict__ in,
                                                       const TA* __restrict__ w, int64_t w_gs,
                                                       float* __restrict__ y, int B, int Hin,
                                                       int Win, int Cin, int Hout, int Wout,
                                                       int Cout, int stride) {
  pdl_begin();
  extern __shared__ float ws[];  // [16][9][Cin]
  const int g = blockIdx.z, co0 = blockIdx.y * 16;
  const int nco = min(16, Cout - co0);
  const TA* wg = w + (int64_t)g * w_gs;
  const int KC = 9 * Cin;
  for (int e = threadIdx.x; e < 16 * KC; e += blockDim.x) {
    const int co = e / KC, r = e % KC;
    ws[e] = co < nco ? Elem<TA>::load(wg + (int64_t)(co0 + co) * KC + r) : 0.f;
  }
  __syncthreads();
  const int64_t P = (int64_t)B * Hout * Wout;
  const int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (p >= P) return;
  const int ow = (int)(p % Wout);
  const int oh = (int)((p / Wout) % Hout);
  const int b = (int)(p / ((int64_t)Wout * Hout));
  float acc[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) acc[i] = 0.f;
  const TA* ing = in + (int64_t)g * B * Hin * Win * Cin;
  for (int kh = 0; kh < 3; ++kh) {
    const int ih = oh * stride + kh - 1;
    if (ih < 0 || ih >= Hin) continue;
    for (int kw = 0; kw < 3; ++kw) {
      const int iw = ow * stride + kw - 1;
      if (iw < 0 || iw >= Win) continue;
      const TA* src = ing + (((int64_t)b * Hin + ih) * Win + iw) * Cin;
      const float* wk = ws + (kh * 3 + kw) * Cin;
      for (int ci = 0; ci < Cin; ++ci) {
        const float x = Elem<TA>::load(src + ci);
#pragma unroll
        for (int co = 0; co < 16; ++co) acc[co] = fmaf(x, wk[co * KC + ci], acc[co]);
      }
    }
  }
  float* dst = y + ((int64_t)g * P + p) * Cout + co0;
  for (int co = 0; co < nco; ++co) dst[co] = acc[co];
}

// Data gradient of conv_fwd: dx[g][b][ih][iw][ci] = sum over the taps that reach (ih, iw) of
// sum_co dy[g][b][oh][ow][co] w[g][co][kh][kw][ci], plus (option-A shortcut) the block's
// pre-activation gradient dout * (out > 0) at (ih / s, iw / s, ci) when ih, iw are multiples of s
// and ci < the block's input channels.
template <typename TA>
__global__ void __launch_bounds__(64) conv_dgrad_kernel(
    const TA* __restrict__ dy, const TA* __restrict__ w, int64_t w_gs, float* __restrict__ dx,
    int B, int Hin, int Win, int Cin, int Hout, int Wout, int Cout, int stride,
    const float* __restrict__ dout, const TA* __restrict__ out_act) {
  pdl_begin();
  extern __shared__ float ws[];  // [Cout][9][16]
  const int g = blockIdx.z, ci0 = blockIdx.y * 16;
  const int nci = min(16, Cin - ci0);
  const TA* wg = w + (int64_t)g * w_gs;
  for (int e = threadIdx.x; e < Cout * 9 * 16; e += blockDim.x) {
    const int ci = e % 16, tap = (e / 16) % 9, co = e / 144;
    ws[e] = ci < nci ? Elem<TA>::load(wg + ((int64_t)co * 9 + tap) * Cin + ci0 + ci) : 0.f;
  }
  __syncthreads();
  const int64_t P = (int64_t)B * Hin * Win;
  const int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (p >= P) return;
  const int iw = (int)(p % Win);
  const int ih = (int)((p / Win) % Hin);
  const int b = (int)(p / ((int64_t)Win * Hin));
  float acc[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) acc[i] = 0.f;
  const TA* dyg = dy + (int64_t)g * B * Hout * Wout * Cout;
  for (int kh = 0; kh < 3; ++kh) {
    const int on = ih + 1 - kh;
    if (on < 0 || on % stride) continue;
    const int oh = on / stride;
    if (oh >= Hout) continue;
    for (int kw = 0; kw < 3; ++kw) {
      const int wn = iw + 1 - kw;
      if (wn < 0 || wn % stride) continue;
      const int ow = wn / stride;
      if (ow >= Wout) continue;
      const TA* src = dyg + (((int64_t)b * Hout + oh) * Wout + ow) * Cout;
      const float* wk = ws + (kh * 3 + kw) * 16;
      for (int co = 0; co < Cout; ++co) {
        const float d = Elem<TA>::load(src + co);
#pragma unroll
        for (int ci = 0; ci < 16; ++ci) acc[ci] = fmaf(d, wk[co * 144 + ci], acc[ci]);
      }
    }
  }
  if (dout && ih % stride == 0 && iw % stride == 0) {
    const int64_t e = ((((int64_t)g * B + b) * Hout + ih / stride) * Wout + iw / stride) * Cout;
    for (int ci = 0; ci < nci; ++ci)
      if (Elem<TA>::load(out_act + e + ci0 + ci) > 0.f) acc[ci] += dout[e + ci0 + ci];
  }
  float* dst = dx + ((int64_t)g * P + p) * Cin + ci0;
  for (int ci = 0; ci < nci; ++ci) dst[ci] = acc[ci];
}

// Weight gradient, pass 1: part[g][q][co][j] = sum over the pixels of chunk q of
// dy[p][co] * im2col(in)[p][j], j = (kh 3 + kw) Cin + ci.  Thread (co = t mod 16, j0 = t / 16)
// owns j = j0 + 16 k; pixels are staged kWgradTile at a time in shared memory.
template <typename TA>
__global__ void __launch_bounds__(256) conv_wgrad_partial_kernel(
    const TA* __restrict__ dy, const TA* __restrict__ in, float* __restrict__ part, int B, int Hin,
    int Win, int Cin, int Hout, int Wout, int Cout, int stride, int nq) {
  pdl_begin();
  extern __shared__ float sm[];
  const int J = 9 * Cin;
  float* dys = sm;                     // [kWgradTile][16]
  float* ims = sm + kWgradTile * 16;   // [kWgradTile][J]
  const int g = blockIdx.z, co0 = blockIdx.y * 16, q = blockIdx.x;
  const int co = threadIdx.x & 15, j0 = threadIdx.x >> 4;
  const int64_t P = (int64_t)B * Hout * Wout;
  const int64_t p0 = (int64_t)q * kWgradChunk, p1 = min(P, p0 + kWgradChunk);
  const TA* dyg = dy + (int64_t)g * P * Cout;
  const TA* ing = in + (int64_t)g * B * Hin * Win * Cin;
  float acc[kMaxJ16];
#pragma unroll
  for (int k = 0; k < kMaxJ16; ++k) acc[k] = 0.f;
  for (int64_t pb = p0; pb < p1; pb += kWgradTile) {
    {
      const int pp = threadIdx.x >> 4, c = threadIdx.x & 15;
      const int64_t p = pb + pp;
      dys[pp * 16 + c] = (p < p1 && co0 + c < Cout) ? Elem<TA>::load(dyg + p * Cout + co0 + c) : 0.f;
    }
    for (int e = threadIdx.x; e < kWgradTile * J; e += blockDim.x) {
      const int pp = e / J, j = e % J;
      const int64_t p = pb + pp;
      float v = 0.f;
      if (p < p1) {
        const int tap = j / Cin, ci = j % Cin;
        const int ow = (int)(p % Wout), oh = (int)((p / Wout) % Hout);
        const int b = (int)(p / ((int64_t)Wout * Hout));
        const int ih = oh * stride + tap / 3 - 1, iw = ow * stride + tap % 3 - 1;
        if (ih >= 0 && ih < Hin && iw >= 0 && iw < Win)
          v = Elem<TA>::load(ing + (((int64_t)b * Hin + ih) * Win + iw) * Cin + ci);
      }
      ims[e] = v;
    }
    __syncthreads();
    for (int pp = 0; pp < kWgradTile; ++pp) {
      const float d = dys[pp * 16 + co];
      const float* row = ims + pp * J;
#pragma unroll
      for (int k = 0; k < kMaxJ16; ++k) {
        const int j = j0 + 16 * k;
        if (j < J) acc[k] = fmaf(d, row[j], acc[k]);
      }
    }
    __syncthreads();
  }
  if (co0 + co < Cout) {
    float* dst = part + (((int64_t)g * nq + q) * Cout + co0 + co) * J;
#pragma unroll
    for (int k = 0; k < kMaxJ16; ++k) {
      const int j = j0 + 16 * k;
      if (j < J) dst[j] = acc[k];
    }
  }
}

// Weight gradient, pass 2: G[g][w_off + e] = sum_q part[g][q][e] in chunk order.
__global__ void sum_partials_kernel(const float* __restrict__ part, int nq, int64_t n, int G,
                                    float* __restrict__ out, int64_t out_gs) {
  pdl_begin();
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < (int64_t)G * n; t += stride) {
    const int g = (int)(t / n);
    const int64_t e = t % n;
    const float* p = part + (int64_t)g * nq * n + e;
    float s = 0.f;
    for (int q = 0; q < nq; ++q) s += p[(int64_t)q * n];
    out[(int64_t)g * out_gs + e] = s;
  }
}

// BatchNorm statistics, pass 1: per chunk of pixels, the chunk mean and the sum of squared
// deviations from it (two passes over the chunk), part[g][q][c] = (mean, M2).
__global__ void __launch_bounds__(256) bn_stats_partial_kernel(const float* __restrict__ y,
                                                               int64_t P, int C, int nq, int chunk,
                                                               float* __restrict__ part) {
  pdl_begin();
  __shared__ float red[256];
  __shared__ float mean_s[256];
  const int g = blockIdx.y, q = blockIdx.x;
  const int lanes = blockDim.x / C;
  const int c = threadIdx.x % C, l = threadIdx.x / C;
  const int64_t p0 = (int64_t)q * chunk, p1 = min(P, p0 + chunk);
  const float* yg = y + (int64_t)g * P * C;
  float s = 0.f;
  if (l < lanes)
    for (int64_t p = p0 + l; p < p1; p += lanes) s += yg[p * C + c];
  red[threadIdx.x] = s;
  __syncthreads();
  if (threadIdx.x < C) {
    float t = 0.f;
    for (int i = 0; i < lanes; ++i) t += red[i * C + threadIdx.x];
    mean_s[threadIdx.x] = t / (float)(p1 - p0);
  }
  __syncthreads();
  const float m = mean_s[c];
  float s2 = 0.f;
  if (l < lanes)
    for (int64_t p = p0 + l; p < p1; p += lanes) {
      const float dv = yg[p * C + c] - m;
      s2 = fmaf(dv, dv, s2);
    }
  __syncthreads();
  red[threadIdx.x] = s2;
  __syncthreads();
  if (threadIdx.x < C) {
    float t = 0.f;
    for (int i = 0; i < lanes; ++i) t += red[i * C + threadIdx.x];
    float* dst = part + (((int64_t)g * nq + q) * C + threadIdx.x) * 2;
    dst[0] = mean_s[threadIdx.x];
    dst[1] = t;
  }
}

// The same for C a multiple of 4 (C / 4 dividing 256): thread = (group of 4 channels, pixel lane),
// float4 loads; each pass's lane sums are combined by a fixed-shape tree in shared memory.
__device__ __forceinline__ void tree_sum4(float4* red, int lane, int lanes, int cg, int C4) {
  int span = 1;
  while (span < lanes) span <<= 1;
  for (int st = span >> 1; st > 0; st >>= 1) {
    __syncthreads();
    if (lane < st && lane + st < lanes) {
      float4& a = red[lane * C4 + cg];
      const float4 b = red[(lane + st) * C4 + cg];
      a.x += b.x;
      a.y += b.y;
      a.z += b.z;
      a.w += b.w;
    }
  }
  __syncthreads();
}

__global__ void __launch_bounds__(256) bn_stats_partial_v4_kernel(const float* __restrict__ y,
                                                                  int64_t P, int C, int nq,
                                                                  int chunk,
                                                                  float* __restrict__ part) {
  pdl_begin();
  __shared__ float4 red[256];
  const int g = blockIdx.y, q = blockIdx.x;
  const int C4 = C / 4, lanes = blockDim.x / C4;
  const int cg = threadIdx.x % C4, l = threadIdx.x / C4;
  const int64_t p0 = (int64_t)q * chunk, p1 = min(P, p0 + chunk);
  const float4* yg = reinterpret_cast<const float4*>(y + (int64_t)g * P * C) + cg;
  float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
  if (l < lanes) {
#pragma unroll 4
    for (int64_t p = p0 + l; p < p1; p += lanes) {
      const float4 v = yg[p * C4];
      s.x += v.x;
      s.y += v.y;
      s.z += v.z;
      s.w += v.w;
    }
    red[l * C4 + cg] = s;
  }
  tree_sum4(red, l < lanes ? l : 0x7fffffff, lanes, cg, C4);
  const float inv = 1.0f / (float)(p1 - p0);
  const float4 tot = red[cg];
  const float4 m = make_float4(tot.x * inv, tot.y * inv, tot.z * inv, tot.w * inv);
  __syncthreads();  // everyone has read red[cg] before it is reused
  float4 s2 = make_float4(0.f, 0.f, 0.f, 0.f);
  if (l < lanes) {
#pragma unroll 4
    for (int64_t p = p0 + l; p < p1; p += lanes) {
      const float4 v = yg[p * C4];
      const float dx = v.x - m.x, dy = v.y - m.y, dz = v.z - m.z, dw = v.w - m.w;
      s2.x = fmaf(dx, dx, s2.x);
      s2.y = fmaf(dy, dy, s2.y);
      s2.z = fmaf(dz, dz, s2.z);
      s2.w = fmaf(dw, dw, s2.w);
    }
    red[l * C4 + cg] = s2;
  }
  tree_sum4(red, l < lanes ? l : 0x7fffffff, lanes, cg, C4);
  if (l == 0) {
    const float4 t2 = red[cg];
    float* dst = part + (((int64_t)g * nq + q) * C + 4 * cg) * 2;
    dst[0] = m.x;
    dst[1] = t2.x;
    dst[2] = m.y;
    dst[3] = t2.y;
    dst[4] = m.z;
    dst[5] = t2.z;
    dst[6] = m.w;
    dst[7] = t2.w;
  }
}

// Pass 2: Chan et al.'s pairwise combination of the chunk (count, mean, M2): one warp per
// (replica, channel); lane l combines chunks l, l + 32, ... in order, then a fixed butterfly of
// shuffles combines the lanes.  Biased variance, rstd = 1 / sqrt(var + eps).
__device__ __forceinline__ void chan_merge(float& n, float& mu, float& M2, float nb, float mb,
                                           float M2b) {
  const float nt = n + nb;
  if (nt <= 0.f) return;
  const float delta = mb - mu, f = nb / nt;
  mu = fmaf(delta, f, mu);
  M2 = M2 + M2b + delta * delta * n * f;
  n = nt;
}

__global__ void bn_stats_finalize_kernel(const float* __restrict__ part, int64_t P, int C, int nq,
                                         int chunk, int G, float* __restrict__ mean,
                                         float* __restrict__ rstd) {
  pdl_begin();
  const int wid = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (wid >= G * C) return;
  const int g = wid / C, c = wid % C;
  float n = 0.f, mu = 0.f, M2 = 0.f;
  for (int q = lane; q < nq; q += 32) {
    const float nb = (float)min((int64_t)chunk, P - (int64_t)q * chunk);
    const float* pq = part + (((int64_t)g * nq + q) * C + c) * 2;
    chan_merge(n, mu, M2, nb, pq[0], pq[1]);
  }
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float n2 = __shfl_xor_sync(0xffffffffu, n, o);
    const float m2 = __shfl_xor_sync(0xffffffffu, mu, o);
    const float M22 = __shfl_xor_sync(0xffffffffu, M2, o);
    // both partners combine (lower lane first) so they hold bit-identical results
    float na = n, ma = mu, Ma = M2;
    float nb = n2, mb = m2, Mb = M22;
    if (lane & o) {
      na = n2; ma = m2; Ma = M22;
      nb = n; mb = mu; Mb = M2;
    }
    chan_merge(na, ma, Ma, nb, mb, Mb);
    n = na;
    mu = ma;
    M2 = Ma;
  }
  if (lane == 0) {
    mean[wid] = mu;
    rstd[wid] = 1.0f / sqrtf(M2 / n + kBnEps);
  }
}

// Four consecutive channels of an activation tensor (bf16 or fp32).
template <typename TA>
struct Vec4;
template <>
struct Vec4<float> {
  __device__ __forceinline__ static float4 load(const float* p) {
    return *reinterpret_cast<const float4*>(p);
  }
  __device__ __forceinline__ static void store(float* p, float4 v) {
    *reinterpret_cast<float4*>(p) = v;
  }
};
template <>
struct Vec4<uint16_t> {
  __device__ __forceinline__ static float4 load(const uint16_t* p) {
    const uint2 u = *reinterpret_cast<const uint2*>(p);
    return make_float4(bf2f((uint16_t)(u.x & 0xffff)), bf2f((uint16_t)(u.x >> 16)),
                       bf2f((uint16_t)(u.y & 0xffff)), bf2f((uint16_t)(u.y >> 16)));
  }
  __device__ __forceinline__ static void store(uint16_t* p, float4 v) {
    uint2 o;
    o.x = (uint32_t)f2bf(v.x) | ((uint32_t)f2bf(v.y) << 16);
    o.y = (uint32_t)f2bf(v.z) | ((uint32_t)f2bf(v.w) << 16);
    *reinterpret_cast<uint2*>(p) = o;
  }
};

// out = relu(gamma (y - mean) rstd + beta [+ option-A shortcut of the block input]); one thread
// per pixel and 4 channels (C a multiple of 4, fewer than 2^31 groups of 4).
template <typename TA>
__global__ void bn_act_fwd_kernel(const float* __restrict__ y, const float* __restrict__ mean,
                                  const float* __restrict__ rstd, const float* __restrict__ W,
                                  int64_t g_off, int64_t b_off, int64_t d_gs, int w_g0, int w_gmul,
                                  const TA* __restrict__ sc, int sc_H, int sc_W, int sc_C,
                                  int stride, TA* __restrict__ out, int G, int B, int H, int Wd,
                                  int C) {
  pdl_begin();
  const int C4 = C / 4;
  const int P = B * H * Wd;
  const int n4 = G * P * C4;
  for (int t = blockIdx.x * blockDim.x + threadIdx.x; t < n4; t += gridDim.x * blockDim.x) {
    const int c0 = (t % C4) * 4;
    const int row = t / C4;
    const int g = row / P, pix = row - g * P;
    const float* Wg = W + (int64_t)(w_g0 + g * w_gmul) * d_gs;
    const float4 yv = *reinterpret_cast<const float4*>(y + (int64_t)t * 4);
    const float yy[4] = {yv.x, yv.y, yv.z, yv.w};
    float v[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int c = c0 + i;
      v[i] = Wg[g_off + c] * ((yy[i] - mean[g * C + c]) * rstd[g * C + c]) + Wg[b_off + c];
    }
    if (sc && c0 < sc_C) {
      const int x = pix % Wd, h = (pix / Wd) % H, b = pix / (Wd * H);
      const float4 s4 = Vec4<TA>::load(
          sc + ((((int64_t)g * B + b) * sc_H + h * stride) * sc_W + x * stride) * sc_C + c0);
      v[0] += s4.x;
      v[1] += s4.y;
      v[2] += s4.z;
      v[3] += s4.w;
    }
    Vec4<TA>::store(out + (int64_t)t * 4, make_float4(fmaxf(v[0], 0.f), fmaxf(v[1], 0.f),
                                                      fmaxf(v[2], 0.f), fmaxf(v[3], 0.f)));
  }
}

// The convolution epilogue's statistics partials (count, mean, M2; one per epilogue warp and CTA)
// merged by Chan et al.'s formula: one warp per (replica, channel); lane l merges partials l,
// l + 32, ... in order, then the fixed butterfly of bn_stats_finalize_kernel combines the lanes.
__global__ void bn_merge_partials_kernel(const float4* __restrict__ stats, int nparts, int G, int C,
                                         float* __restrict__ mean, float* __restrict__ rstd) {
  pdl_begin();
  const int wid = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (wid >= G * C) return;
  const int g = wid / C, c = wid % C;
  const float4* src = stats + (int64_t)g * nparts * C + c;
  float n = 0.f, mu = 0.f, M2 = 0.f;
  for (int q = lane; q < nparts; q += 32) {
    const float4 v = __ldg(src + (int64_t)q * C);
    chan_merge(n, mu, M2, v.x, v.y, v.z);
  }
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float n2 = __shfl_xor_sync(0xffffffffu, n, o);
    const float m2 = __shfl_xor_sync(0xffffffffu, mu, o);
    const float M22 = __shfl_xor_sync(0xffffffffu, M2, o);
    // both partners combine (lower lane first) so they hold bit-identical results
    float na = n, ma = mu, Ma = M2;
    float nb = n2, mb = m2, Mb = M22;
    if (lane & o) {
      na = n2; ma = m2; Ma = M22;
      nb = n; mb = mu; Mb = M2;
    }
    chan_merge(na, ma, Ma, nb, mb, Mb);
    n = na;
    mu = ma;
    M2 = Ma;
  }
  if (lane == 0) {
    mean[wid] = mu;
    rstd[wid] = 1.0f / sqrtf(M2 / n + kBnEps);
  }
}

// The same with a fixed group of 4 channels per thread (C / 4 dividing the block size): the
// channels' gamma, beta, mean and rstd are loaded once, pixels advance by grid strides, and the
// replica is blockIdx.y (32-bit pixel indexing).
template <typename TA>
__global__ void __launch_bounds__(256) bn_act_fwd_v4_kernel(
    const float* __restrict__ y, const float* __restrict__ mean, const float* __restrict__ rstd,
    const float* __restrict__ W, int64_t g_off, int64_t b_off, int64_t d_gs, int w_g0, int w_gmul,
    const TA* __restrict__ sc, int sc_H, int sc_W, int sc_C, int stride, TA* __restrict__ out, int B,
    int H, int Wd, int C) {
  pdl_begin();
  const int g = blockIdx.y, C4 = C / 4;
  const int c0 = (threadIdx.x % C4) * 4, pl = threadIdx.x / C4, ppb = blockDim.x / C4;
  const int P = B * H * Wd;
  const float* Wg = W + (int64_t)(w_g0 + g * w_gmul) * d_gs;
  float ga[4], be[4], mu[4], rs[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    ga[i] = Wg[g_off + c0 + i];
    be[i] = Wg[b_off + c0 + i];
    mu[i] = mean[g * C + c0 + i];
    rs[i] = rstd[g * C + c0 + i];
  }
  const bool with_sc = sc && c0 < sc_C;
  // identity shortcut (same grid): the shortcut pixel is p itself, no index arithmetic per pixel
  const bool sc_same = stride == 1 && sc_H == H && sc_W == Wd;
  const float* yg = y + (int64_t)g * P * C + c0;
  TA* og = out + (int64_t)g * P * C + c0;
  for (int p = blockIdx.x * ppb + pl; p < P; p += gridDim.x * ppb) {
    const float4 yv = *reinterpret_cast<const float4*>(yg + (int64_t)p * C);
    float4 s4 = make_float4(0.f, 0.f, 0.f, 0.f);
    if (with_sc) {
      int64_t sp;
      if (sc_same) {
        sp = (int64_t)g * P + p;
      } else {
        const int x = p % Wd, hb = p / Wd, h = hb % H, b = hb / H;
        sp = (((int64_t)g * B + b) * sc_H + h * stride) * sc_W + x * stride;
      }
      s4 = Vec4<TA>::load(sc + sp * sc_C + c0);
    }
    const float yy[4] = {yv.x, yv.y, yv.z, yv.w};
    float v[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) v[i] = ga[i] * ((yy[i] - mu[i]) * rs[i]) + be[i];
    if (with_sc) {
      v[0] += s4.x;
      v[1] += s4.y;
      v[2] += s4.z;
      v[3] += s4.w;
    }
    Vec4<TA>::store(og + (int64_t)p * C, make_float4(fmaxf(v[0], 0.f), fmaxf(v[1], 0.f),
                                                    fmaxf(v[2], 0.f), fmaxf(v[3], 0.f)));
  }
}

// BatchNorm backward, pass 1: with dz = dout * (out > 0) and xhat = (y - mean) rstd, chunk sums
// part[g][q][c] = (sum dz, sum dz xhat).
template <typename TA>
__global__ void __launch_bounds__(256) bn_bwd_partial_kernel(
    const float* __restrict__ dout, const TA* __restrict__ out, const float* __restrict__ y,
    const float* __restrict__ mean, const float* __restrict__ rstd, int64_t P, int C, int nq,
    int chunk, float* __restrict__ part) {
  pdl_begin();
  __shared__ float r1[256], r2[256];
  const int g = blockIdx.y, q = blockIdx.x;
  const int lanes = blockDim.x / C;
  const int c = threadIdx.x % C, l = threadIdx.x / C;
  const int64_t p0 = (int64_t)q * chunk, p1 = min(P, p0 + chunk);
  const int64_t base = (int64_t)g * P * C;
  const float mu = mean[g * C + c], rs = rstd[g * C + c];
  float s1 = 0.f, s2 = 0.f;
  if (l < lanes)
#pragma unroll 4
    for (int64_t p = p0 + l; p < p1; p += lanes) {
      const int64_t e = base + p * C + c;
      const float dz = Elem<TA>::load(out + e) > 0.f ? dout[e] : 0.f;
      s1 += dz;
      s2 = fmaf(dz, (y[e] - mu) * rs, s2);
    }
  r1[threadIdx.x] = s1;
  r2[threadIdx.x] = s2;
  __syncthreads();
  if (threadIdx.x < C) {
    float t1 = 0.f, t2 = 0.f;
    for (int i = 0; i < lanes; ++i) {
      t1 += r1[i * C + threadIdx.x];
      t2 += r2[i * C + threadIdx.x];
    }
    float* dst = part + (((int64_t)g * nq + q) * C + threadIdx.x) * 2;
    dst[0] = t1;
    dst[1] = t2;
  }
}

// The same for C a multiple of 4 (C / 4 dividing 256), float4 / 4-channel loads and a fixed-shape
// tree over the pixel lanes.
template <typename TA>
__global__ void __launch_bounds__(256) bn_bwd_partial_v4_kernel(
    const float* __restrict__ dout, const TA* __restrict__ out, const float* __restrict__ y,
    const float* __restrict__ mean, const float* __restrict__ rstd, int64_t P, int C, int nq,
    int chunk, float* __restrict__ part) {
  pdl_begin();
  __shared__ float4 r1[256], r2[256];
  const int g = blockIdx.y, q = blockIdx.x;
  const int C4 = C / 4, lanes = blockDim.x / C4;
  const int cg = threadIdx.x % C4, l = threadIdx.x / C4;
  const int64_t p0 = (int64_t)q * chunk, p1 = min(P, p0 + chunk);
  const int64_t base = (int64_t)g * P * C + 4 * cg;
  const float4 mu = *reinterpret_cast<const float4*>(mean + g * C + 4 * cg);
  const float4 rs = *reinterpret_cast<const float4*>(rstd + g * C + 4 * cg);
  float4 s1 = make_float4(0.f, 0.f, 0.f, 0.f), s2 = s1;
  if (l < lanes) {
#pragma unroll 4
    for (int64_t p = p0 + l; p < p1; p += lanes) {
      const int64_t e = base + p * C;
      const float4 d = *reinterpret_cast<const float4*>(dout + e);
      const float4 o = Vec4<TA>::load(out + e);
      const float4 v = *reinterpret_cast<const float4*>(y + e);
      const float dz0 = o.x > 0.f ? d.x : 0.f, dz1 = o.y > 0.f ? d.y : 0.f;
      const float dz2 = o.z > 0.f ? d.z : 0.f, dz3 = o.w > 0.f ? d.w : 0.f;
      s1.x += dz0;
      s1.y += dz1;
      s1.z += dz2;
      s1.w += dz3;
      s2.x = fmaf(dz0, (v.x - mu.x) * rs.x, s2.x);
      s2.y = fmaf(dz1, (v.y - mu.y) * rs.y, s2.y);
      s2.z = fmaf(dz2, (v.z - mu.z) * rs.z, s2.z);
      s2.w = fmaf(dz3, (v.w - mu.w) * rs.w, s2.w);
    }
    r1[l * C4 + cg] = s1;
    r2[l * C4 + cg] = s2;
  }
  int span = 1;
  while (span < lanes) span <<= 1;
  for (int st = span >> 1; st > 0; st >>= 1) {
    __syncthreads();
    if (l < st && l + st < lanes) {
      float4& a = r1[l * C4 + cg];
      const float4 b = r1[(l + st) * C4 + cg];
      a.x += b.x;
      a.y += b.y;
      a.z += b.z;
      a.w += b.w;
      float4& a2 = r2[l * C4 + cg];
      const float4 b2 = r2[(l + st) * C4 + cg];
      a2.x += b2.x;
      a2.y += b2.y;
      a2.z += b2.z;
      a2.w += b2.w;
    }
  }
  __syncthreads();
  if (l == 0) {
    const float4 t1 = r1[cg], t2 = r2[cg];
    float* dst = part + (((int64_t)g * nq + q) * C + 4 * cg) * 2;
    dst[0] = t1.x;
    dst[1] = t2.x;
    dst[2] = t1.y;
    dst[3] = t2.y;
    dst[4] = t1.z;
    dst[5] = t2.z;
    dst[6] = t1.w;
    dst[7] = t2.w;
  }
}

// Pass 2: s[g][c] = the chunk sums (one warp per (replica, channel): lane l adds chunks l, l + 32,
// ... in order, then a fixed butterfly); dgamma = sum dz xhat, dbeta = sum dz into G.
__global__ void bn_bwd_finalize_kernel(const float* __restrict__ part, int C, int nq, int G,
                                       float* __restrict__ s12, float* __restrict__ Gr,
                                       int64_t g_off, int64_t b_off, int64_t d_gs) {
  pdl_begin();
  const int wid = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (wid >= G * C) return;
  const int g = wid / C, c = wid % C;
  float a = 0.f, b = 0.f;
  for (int q = lane; q < nq; q += 32) {
    const float* pq = part + (((int64_t)g * nq + q) * C + c) * 2;
    a += pq[0];
    b += pq[1];
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    a += __shfl_xor_sync(0xffffffffu, a, o);
    b += __shfl_xor_sync(0xffffffffu, b, o);
  }
  if (lane == 0) {
    s12[(int64_t)wid * 2] = a;
    s12[(int64_t)wid * 2 + 1] = b;
    Gr[(int64_t)g * d_gs + g_off + c] = b;
    Gr[(int64_t)g * d_gs + b_off + c] = a;
  }
}

// The same sums from the data-gradient convolution's epilogue partials (ConvBwdFuse): one warp
// per (replica, channel); lane l adds partials l, l + 32, ... in order, then a fixed butterfly.
__global__ void bn_bwd_merge_kernel(const float2* __restrict__ part, int nparts, int C, int G,
                                    float* __restrict__ s12, float* __restrict__ Gr, int64_t g_off,
                                    int64_t b_off, int64_t d_gs) {
  pdl_begin();
  const int wid = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (wid >= G * C) return;
  const int g = wid / C, c = wid % C;
  float a = 0.f, b = 0.f;
  for (int q = lane; q < nparts; q += 32) {
    const float2 v = part[((int64_t)g * nparts + q) * C + c];
    a += v.x;
    b += v.y;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    a += __shfl_xor_sync(0xffffffffu, a, o);
    b += __shfl_xor_sync(0xffffffffu, b, o);
  }
  if (lane == 0) {
    s12[(int64_t)wid * 2] = a;
    s12[(int64_t)wid * 2 + 1] = b;
    Gr[(int64_t)g * d_gs + g_off + c] = b;
    Gr[(int64_t)g * d_gs + b_off + c] = a;
  }
}

// dy = gamma rstd (dz - mean(dz) - xhat mean(dz xhat)), the convolution's output gradient; one
// thread per pixel and 4 channels.
template <typename TA>
__global__ void bn_bwd_apply_kernel(const float* __restrict__ dout, const TA* __restrict__ out,
                                    const float* __restrict__ y, const float* __restrict__ mean,
                                    const float* __restrict__ rstd, const float* __restrict__ s12,
                                    const float* __restrict__ W, int64_t g_off, int64_t d_gs,
                                    TA* __restrict__ dy, int G, int64_t P64, int C) {
  pdl_begin();
  const int C4 = C / 4;
  const int P = (int)P64;
  const int n4 = G * P * C4;
  const float invM = 1.0f / (float)P;
  for (int t = blockIdx.x * blockDim.x + threadIdx.x; t < n4; t += gridDim.x * blockDim.x) {
    const int c0 = (t % C4) * 4;
    const int g = (t / C4) / P;
    const float4 d4 = *reinterpret_cast<const float4*>(dout + (int64_t)t * 4);
    const float4 o4 = Vec4<TA>::load(out + (int64_t)t * 4);
    const float4 y4 = *reinterpret_cast<const float4*>(y + (int64_t)t * 4);
    const float dd[4] = {d4.x, d4.y, d4.z, d4.w}, oo[4] = {o4.x, o4.y, o4.z, o4.w};
    const float yy[4] = {y4.x, y4.y, y4.z, y4.w};
    float v[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int gc = g * C + c0 + i;
      const float dz = oo[i] > 0.f ? dd[i] : 0.f;
      const float xh = (yy[i] - mean[gc]) * rstd[gc];
      v[i] = W[(int64_t)g * d_gs + g_off + c0 + i] * rstd[gc] *
             (dz - s12[2 * gc] * invM - xh * (s12[2 * gc + 1] * invM));
    }
    Vec4<TA>::store(dy + (int64_t)t * 4, make_float4(v[0], v[1], v[2], v[3]));
  }
}

// The same with a fixed group of 4 channels per thread (C / 4 dividing the block size), the
// per-channel factors loaded once, blockIdx.y the replica.  out == nullptr: dout is already
// masked (the data-gradient epilogue applied the ReLU), so dz = dout.
template <typename TA>
__global__ void __launch_bounds__(256) bn_bwd_apply_v4_kernel(
    const float* __restrict__ dout, const TA* __restrict__ out, const float* __restrict__ y,
    const float* __restrict__ mean, const float* __restrict__ rstd, const float* __restrict__ s12,
    const float* __restrict__ W, int64_t g_off, int64_t d_gs, TA* __restrict__ dy, int P, int C) {
  pdl_begin();
  const int g = blockIdx.y, C4 = C / 4;
  const int c0 = (threadIdx.x % C4) * 4, pl = threadIdx.x / C4, ppb = blockDim.x / C4;
  const float invM = 1.0f / (float)P;
  float mu[4], rs[4], gr[4], m1[4], m2[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int gc = g * C + c0 + i;
    mu[i] = mean[gc];
    rs[i] = rstd[gc];
    gr[i] = W[(int64_t)g * d_gs + g_off + c0 + i] * rs[i];
    m1[i] = s12[2 * gc] * invM;
    m2[i] = s12[2 * gc + 1] * invM;
  }
  const int64_t base = (int64_t)g * P * C + c0;
  for (int p = blockIdx.x * ppb + pl; p < P; p += gridDim.x * ppb) {
    const int64_t e = base + (int64_t)p * C;
    const float4 d4 = *reinterpret_cast<const float4*>(dout + e);
    const float4 o4 = out ? Vec4<TA>::load(out + e) : make_float4(1.f, 1.f, 1.f, 1.f);
    const float4 y4 = *reinterpret_cast<const float4*>(y + e);
    const float dd[4] = {d4.x, d4.y, d4.z, d4.w}, oo[4] = {o4.x, o4.y, o4.z, o4.w};
    const float yy[4] = {y4.x, y4.y, y4.z, y4.w};
    float v[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float dz = oo[i] > 0.f ? dd[i] : 0.f;
      const float xh = (yy[i] - mu[i]) * rs[i];
      v[i] = gr[i] * (dz - m1[i] - xh * m2[i]);
    }
    Vec4<TA>::store(dy + e, make_float4(v[0], v[1], v[2], v[3]));
  }
}

// feat[g][b][f] = mean over the H W pixels of act[g][b][.][.][f].
template <typename TA>
__global__ void avgpool_kernel(const TA* __restrict__ act, float* __restrict__ feat, int GB, int HW,
                               int F) {
  pdl_begin();
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= GB * F) return;
  const int gb = t / F, f = t % F;
  const TA* src = act + (int64_t)gb * HW * F + f;
  float s = 0.f;
  for (int p = 0; p < HW; ++p) s += Elem<TA>::load(src + (int64_t)p * F);
  feat[t] = s / (float)HW;
}

// dact[g][b][p][f] = dfeat[g][b][f] / HW (gradient of the average pooling).
__global__ void avgpool_bwd_kernel(const float* __restrict__ dfeat, float* __restrict__ dact,
                                   int64_t n, int HW, int F) {
  pdl_begin();
  const int64_t step = (int64_t)gridDim.x * blockDim.x;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n; e += step) {
    const int f = (int)(e % F);
    const int64_t gb = e / ((int64_t)HW * F);
    dact[e] = dfeat[gb * F + f] / (float)HW;
  }
}

// im2col for the tensor-core convolutions: col[g][p][(kh 3 + kw) Cin + ci] =
// in[g][b][oh s + kh - 1][ow s + kw - 1][ci] (zero outside the image), p = (b, oh, ow); bf16, Cin a
// multiple of 8.  blockIdx.y is the replica; thread e of the replica takes pixel e / R and 16-byte
// chunk e % R of its column row (R = 9 Cin / 8), so consecutive threads write consecutive chunks.
__global__ void __launch_bounds__(256) im2col_v2_kernel(const uint16_t* __restrict__ in,
                                                        uint16_t* __restrict__ col, int B, int Hin,
                                                        int Win, int Cin, int Hout, int Wout,
                                                        int stride) {
  pdl_begin();
  const int g = blockIdx.y, c8n = Cin / 8, R = 9 * c8n;
  const int P = B * Hout * Wout;
  const int e = blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= P * R) return;
  const int p = e / R, r = e - p * R;
  const int tap = r / c8n, c8 = r - tap * c8n;
  const int ow = p % Wout, t2 = p / Wout, oh = t2 % Hout, b = t2 / Hout;
  const int ih = oh * stride + tap / 3 - 1, iw = ow * stride + tap % 3 - 1;
  uint4 v = make_uint4(0u, 0u, 0u, 0u);
  if (ih >= 0 && ih < Hin && iw >= 0 && iw < Win)
    v = __ldg(reinterpret_cast<const uint4*>(
        in + ((((int64_t)g * B + b) * Hin + ih) * Win + iw) * Cin + c8 * 8));
  *reinterpret_cast<uint4*>(col + ((int64_t)g * P + p) * 9 * Cin + (int64_t)r * 8) = v;
}

// The same with the channel count a template constant: a CTA per output row (b, oh) of replica
// blockIdx.y, its threads over the row's Wout x 9 Cin / 8 chunks (divisions by constants only).
template <int C8N>
__global__ void __launch_bounds__(256) im2col_row_kernel(const uint16_t* __restrict__ in,
                                                         uint16_t* __restrict__ col, int B, int Hin,
                                                         int Win, int Hout, int Wout, int stride) {
  pdl_begin();
  constexpr int Cin = 8 * C8N, R = 9 * C8N;
  const int g = blockIdx.y, row = blockIdx.x;
  const int oh = row % Hout, b = row / Hout;
  const int64_t P = (int64_t)B * Hout * Wout;
  const uint16_t* ing = in + ((int64_t)g * B + b) * Hin * Win * Cin;
  uint16_t* out = col + ((int64_t)g * P + (int64_t)row * Wout) * 9 * Cin;
  for (int e = threadIdx.x; e < Wout * R; e += blockDim.x) {
    const int ow = e / R, r = e - ow * R;
    const int tap = r / C8N, c8 = r - tap * C8N;
    const int ih = oh * stride + tap / 3 - 1, iw = ow * stride + tap % 3 - 1;
    uint4 v = make_uint4(0u, 0u, 0u, 0u);
    if (ih >= 0 && ih < Hin && iw >= 0 && iw < Win)
      v = __ldg(reinterpret_cast<const uint4*>(ing + ((int64_t)ih * Win + iw) * Cin + c8 * 8));
    *reinterpret_cast<uint4*>(out + (int64_t)e * 8) = v;
  }
}

// im2col with any channel count, one CTA per output row (b, oh) of replica blockIdx.y: its
// threads over the row's Wout x ldc column entries (32-bit indexing).
template <typename TA>
__global__ void __launch_bounds__(256) im2col_any_row_kernel(const TA* __restrict__ in,
                                                             uint16_t* __restrict__ col, int B,
                                                             int Hin, int Win, int Cin, int Hout,
                                                             int Wout, int stride, int ldc) {
  pdl_begin();
  const int g = blockIdx.y, row = blockIdx.x;
  const int oh = row % Hout, b = row / Hout;
  const int64_t P = (int64_t)B * Hout * Wout;
  const TA* ing = in + ((int64_t)g * B + b) * Hin * Win * Cin;
  uint16_t* out = col + ((int64_t)g * P + (int64_t)row * Wout) * ldc;
  const int J = 9 * Cin;
  for (int e = threadIdx.x; e < Wout * ldc; e += blockDim.x) {
    const int ow = e / ldc, j = e - ow * ldc;
    float v = 0.f;
    if (j < J) {
      const int tap = j / Cin, ci = j - tap * Cin;
      const int ih = oh * stride + tap / 3 - 1, iw = ow * stride + tap % 3 - 1;
      if (ih >= 0 && ih < Hin && iw >= 0 && iw < Win)
        v = Elem<TA>::load(ing + (ih * Win + iw) * Cin + ci);
    }
    out[e] = f2bf(v);
  }
}

// Column matrix of a data gradient: for each pixel (ih, iw) of the convolution's input and each
// flipped tap t' = (kh', kw'), the output-gradient row at ((ih + kh' - 1) / s, (iw + kw' - 1) / s)
// when both are whole and inside the output, else zero.  With the flipped, transposed weights
// this writes dx = sum over the taps reaching (ih, iw) of dy w (stride 1 or 2).  blockIdx.y is
// the replica; thread = (pixel, 16-byte chunk), 32-bit indexing.
__global__ void __launch_bounds__(256) col_dgrad_v2_kernel(const uint16_t* __restrict__ dy,
                                                           uint16_t* __restrict__ col, int B, int Hin,
                                                           int Win, int Cout, int Hout, int Wout,
                                                           int stride) {
  pdl_begin();
  const int g = blockIdx.y, c8n = Cout / 8, R = 9 * c8n;
  const int P = B * Hin * Win;
  const int e = blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= P * R) return;
  const int p = e / R, r = e - p * R;
  const int tap = r / c8n, c8 = r - tap * c8n;
  const int iw = p % Win, t2 = p / Win, ih = t2 % Hin, b = t2 / Hin;
  const int hn = ih + tap / 3 - 1, wn = iw + tap % 3 - 1;
  uint4 v = make_uint4(0u, 0u, 0u, 0u);
  if (hn >= 0 && wn >= 0 && hn % stride == 0 && wn % stride == 0 && hn / stride < Hout &&
      wn / stride < Wout)
    v = __ldg(reinterpret_cast<const uint4*>(
        dy + ((((int64_t)g * B + b) * Hout + hn / stride) * Wout + wn / stride) * Cout + c8 * 8));
  *reinterpret_cast<uint4*>(col + ((int64_t)g * P + p) * 9 * Cout + (int64_t)r * 8) = v;
}

// The same as one CTA per input row (b, ih) of replica blockIdx.y, the output-gradient channel
// count a template constant.
template <int C8N>
__global__ void __launch_bounds__(256) col_dgrad_row_kernel(const uint16_t* __restrict__ dy,
                                                            uint16_t* __restrict__ col, int B,
                                                            int Hin, int Win, int Hout, int Wout,
                                                            int stride) {
  pdl_begin();
  constexpr int Cout = 8 * C8N, R = 9 * C8N;
  const int g = blockIdx.y, row = blockIdx.x;
  const int ih = row % Hin, b = row / Hin;
  const int64_t P = (int64_t)B * Hin * Win;
  const uint16_t* dyg = dy + ((int64_t)g * B + b) * Hout * Wout * Cout;
  uint16_t* out = col + ((int64_t)g * P + (int64_t)row * Win) * 9 * Cout;
  for (int e = threadIdx.x; e < Win * R; e += blockDim.x) {
    const int iw = e / R, r = e - iw * R;
    const int tap = r / C8N, c8 = r - tap * C8N;
    const int hn = ih + tap / 3 - 1, wn = iw + tap % 3 - 1;
    uint4 v = make_uint4(0u, 0u, 0u, 0u);
    if (hn >= 0 && wn >= 0 && hn % stride == 0 && wn % stride == 0 && hn / stride < Hout &&
        wn / stride < Wout)
      v = __ldg(reinterpret_cast<const uint4*>(dyg + ((hn / stride) * Wout + wn / stride) * Cout +
                                               c8 * 8));
    *reinterpret_cast<uint4*>(out + (int64_t)e * 8) = v;
  }
}

// Weights with each [9 Cin] row padded to ldc columns (zeros), bf16: the stem's tensor-core
// operand (9 Cin = 27 is not a multiple of 8).
__global__ void pad_weights_kernel(const uint16_t* __restrict__ Wb, int64_t d_pad, int64_t w_off,
                                   uint16_t* __restrict__ out, int G, int rows, int cols, int ldc) {
  pdl_begin();
  const int64_t n = (int64_t)G * rows * ldc;
  const int64_t step = (int64_t)gridDim.x * blockDim.x;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n; e += step) {
    const int j = (int)(e % ldc);
    const int r = (int)((e / ldc) % rows);
    const int g = (int)(e / ((int64_t)rows * ldc));
    out[e] = j < cols ? Wb[(int64_t)g * d_pad + w_off + (int64_t)r * cols + j] : (uint16_t)0;
  }
}

// Sum of split partials [g][q][rows][ldc] in split order, keeping the first `cols` columns:
// out[g * out_gs + r cols + j].
// out[g out_gs + r cols + j] = sum over q of part[g][q][r][src(j)] (j < cols of ldc), src(j) = j,
// or with taps of tap_dst channels read from taps of tap_src channels (a padded convolution's
// weight gradient cropped to its real input channels): src(j) = (j / tap_dst) tap_src + j % tap_dst.
// A CTA takes 32 consecutive outputs (one per lane); warp w sums the partials q = w, w + 8, ...
// (independent loads, all in flight), and the eight warp sums are added in warp order: a fixed
// order, so the result is deterministic.
constexpr int kSumWarps = 8;
__global__ void __launch_bounds__(32 * kSumWarps) sum_partials_crop_kernel(
    const float* __restrict__ part, int nq, int rows, int ldc, int cols, int G,
    float* __restrict__ out, int64_t out_gs, int tap_src, int tap_dst) {
  pdl_begin();
  __shared__ float ws[kSumWarps][32];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t n = (int64_t)G * rows * cols;
  const int64_t t = (int64_t)blockIdx.x * 32 + lane;
  float acc = 0.f;
  int g = 0, r = 0, j = 0;
  if (t < n) {
    j = (int)(t % cols);
    r = (int)((t / cols) % rows);
    g = (int)(t / ((int64_t)rows * cols));
    const int js = tap_dst > 0 ? (j / tap_dst) * tap_src + j % tap_dst : j;
    const float* p = part + (int64_t)g * nq * rows * ldc + (int64_t)r * ldc + js;
    const int64_t qs = (int64_t)rows * ldc;
#pragma unroll 4
    for (int q = warp; q < nq; q += kSumWarps) acc += p[q * qs];
  }
  ws[warp][lane] = acc;
  __syncthreads();
  if (warp == 0 && t < n) {
    float sum = 0.f;
#pragma unroll
    for (int w = 0; w < kSumWarps; ++w) sum += ws[w][lane];
    out[(int64_t)g * out_gs + (int64_t)r * cols + j] = sum;
  }
}
unsigned sum_partials_grid(int64_t n) { return (unsigned)((n + 31) / 32); }

// The same sum for four consecutive outputs per thread (float4 loads and store), partials added in
// split order q = 0, 1, ...: for column counts, leading dimensions, tap widths and destinations
// that keep every group of four outputs contiguous and 16-byte aligned (sum_partials_v4_ok).
__global__ void __launch_bounds__(256) sum_partials_v4_kernel(
    const float* __restrict__ part, int nq, int rows, int ldc, int cols, int G,
    float* __restrict__ out, int64_t out_gs, int tap_src, int tap_dst) {
  pdl_begin();
  const int64_t n4 = (int64_t)G * rows * (cols / 4);
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= n4) return;
  const int j = (int)(t % (cols / 4)) * 4;
  const int r = (int)((t / (cols / 4)) % rows);
  const int g = (int)(t / ((int64_t)rows * (cols / 4)));
  const int js = tap_dst > 0 ? (j / tap_dst) * tap_src + j % tap_dst : j;
  const float* p = part + (int64_t)g * nq * rows * ldc + (int64_t)r * ldc + js;
  const int64_t qs = (int64_t)rows * ldc;
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
  for (int q = 0; q < nq; ++q) {
    const float4 v = __ldg(reinterpret_cast<const float4*>(p + q * qs));
    acc.x += v.x;
    acc.y += v.y;
    acc.z += v.z;
    acc.w += v.w;
  }
  *reinterpret_cast<float4*>(out + (int64_t)g * out_gs + (int64_t)r * cols + j) = acc;
}

bool sum_partials_v4_ok(const float* part, int ldc, int cols, const float* out, int64_t out_gs,
                        int tap_src, int tap_dst) {
  return cols % 4 == 0 && ldc % 4 == 0 && out_gs % 4 == 0 &&
         (tap_dst == 0 || (tap_dst % 4 == 0 && tap_src % 4 == 0)) &&
         (reinterpret_cast<uintptr_t>(part) & 15) == 0 && (reinterpret_cast<uintptr_t>(out) & 15) == 0;
}

// Several weight gradients' partial sums in one launch (the ResNet step's, at the end of its
// backward): job k covers threads [begin_k, begin_{k+1}) and is sum_partials_v4_kernel's sum for
// its buffers, partials added in split order q = 0, 1, ... -- the same bits as one launch each.
struct SumJob {
  const float* part;
  float* out;
  int64_t out_gs;
  int64_t begin;  // first thread of this job
  int nq, rows, ldc, cols, G, tap_src, tap_dst, pad;
};
constexpr int kMaxSumJobs = 24;
struct SumJobs {
  int n;
  SumJob j[kMaxSumJobs];
};

__global__ void __launch_bounds__(256) sum_partials_jobs_v4_kernel(const __grid_constant__ SumJobs js,
                                                                     int64_t total) {
  pdl_begin();
  const int64_t t0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t0 >= total) return;
  int k = 0;
  while (k + 1 < js.n && t0 >= js.j[k + 1].begin) ++k;
  const SumJob& jb = js.j[k];
  const int64_t t = t0 - jb.begin;
  const int c4 = jb.cols / 4;
  const int j = (int)(t % c4) * 4;
  const int r = (int)((t / c4) % jb.rows);
  const int g = (int)(t / ((int64_t)jb.rows * c4));
  const int js_ = jb.tap_dst > 0 ? (j / jb.tap_dst) * jb.tap_src + j % jb.tap_dst : j;
  const float* pp = jb.part + (int64_t)g * jb.nq * jb.rows * jb.ldc + (int64_t)r * jb.ldc + js_;
  const int64_t qs = (int64_t)jb.rows * jb.ldc;
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
  for (int q = 0; q < jb.nq; ++q) {
    const float4 v = __ldg(reinterpret_cast<const float4*>(pp + q * qs));
    acc.x += v.x;
    acc.y += v.y;
    acc.z += v.z;
    acc.w += v.w;
  }
  *reinterpret_cast<float4*>(jb.out + (int64_t)g * jb.out_gs + (int64_t)r * jb.cols + j) = acc;
}

// Launches whichever of the two partial-sum kernels fits the shapes.
void launch_sum_partials(const float* part, int nq, int rows, int ldc, int cols, int G, float* out,
                         int64_t out_gs, int tap_src, int tap_dst, cudaStream_t s) {
  if (sum_partials_v4_ok(part, ldc, cols, out, out_gs, tap_src, tap_dst)) {
    const int64_t n4 = (int64_t)G * rows * (cols / 4);
    launch_pdl(sum_partials_v4_kernel, (unsigned)((n4 + 255) / 256), 256, 0, s, part, nq, rows, ldc,
               cols, G, out, out_gs, tap_src, tap_dst);
  } else {
    launch_pdl(sum_partials_crop_kernel, sum_partials_grid((int64_t)G * rows * cols),
               32 * kSumWarps, 0, s, part, nq, rows, ldc, cols, G, out, out_gs, tap_src, tap_dst);
  }
}

// The stem's image with zero channels appended: x16[q][c] = c < C0 ? x0[q][c] : 0 (one thread per
// pixel, two 16-byte stores).
__global__ void pad_input16_kernel(const uint16_t* __restrict__ x0, uint16_t* __restrict__ x16,
                                   int64_t npix, int C0) {
  pdl_begin();
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < npix; q += stride) {
    uint32_t w[8] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
    for (int c = 0; c < C0; ++c) w[c >> 1] |= (uint32_t)x0[q * C0 + c] << (16 * (c & 1));
    uint4* dst = reinterpret_cast<uint4*>(x16 + q * 16);
    dst[0] = make_uint4(w[0], w[1], w[2], w[3]);
    dst[1] = make_uint4(w[4], w[5], w[6], w[7]);
  }
}

// The stem's weights with the same zero channels: wstem[g][co][t][ci] = ci < C0 ?
// W[g][co][t][ci] : 0 (bf16, 16 channels per tap).
__global__ void pad_stem_weights_kernel(const uint16_t* __restrict__ Wb, int64_t d_pad,
                                        int64_t w_off, uint16_t* __restrict__ wstem, int G,
                                        int Cout, int C0) {
  pdl_begin();
  const int64_t n = (int64_t)G * Cout * 9 * 16;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n; e += stride) {
    const int ci = (int)(e % 16), t = (int)((e / 16) % 9), co = (int)((e / 144) % Cout);
    const int64_t g = e / (144 * (int64_t)Cout);
    wstem[e] = ci < C0 ? Wb[g * d_pad + w_off + ((int64_t)co * 9 + t) * C0 + ci] : (uint16_t)0;
  }
}

// Weights of the stride-1 data gradient as a convolution of the output gradient:
// wt[g][ci][t][co] = w[g][co][8 - t][ci] (taps flipped, channels transposed), bf16.
__global__ void flip_weights_kernel(const uint16_t* __restrict__ Wb, int64_t d_pad, int64_t w_off,
                                    uint16_t* __restrict__ wt, int G, int Cin, int Cout) {
  pdl_begin();
  // blockIdx.y = replica; 32-bit indexing within it (Cin 9 Cout < 2^31)
  const int g = blockIdx.y, n = Cin * 9 * Cout;
  const uint16_t* src = Wb + (int64_t)g * d_pad + w_off;
  uint16_t* dst = wt + (int64_t)g * n;
  for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < n; e += gridDim.x * blockDim.x) {
    const int co = e % Cout, t = (e / Cout) % 9, ci = e / (9 * Cout);
    dst[e] = src[(co * 9 + (8 - t)) * Cin + ci];
  }
}

// The data gradient of a stride-2 convolution split by the parity (py, px) of the input pixel:
// dx[2a + py][2b + px][ci] = sum over dr, dc in {0, 1} and co of dy[a + dr][b + dc][co]
// w[co][py + 1 - 2 dr][px + 1 - 2 dc][ci] (terms whose kernel index leaves 0..2 drop out), a
// 3x3 stride-1 convolution of dy whose taps (dr + 1, dc + 1) carry those weights and whose other
// taps are zero.  wt4[ph][g][ci][t][co], ph = 2 py + px, t = 3 (dr + 1) + (dc + 1).
__global__ void flip_phase_weights_kernel(const uint16_t* __restrict__ Wb, int64_t d_pad,
                                          int64_t w_off, uint16_t* __restrict__ wt4, int G,
                                          int Cin, int Cout) {
  pdl_begin();
  const int64_t per = (int64_t)Cin * 9 * Cout, n = 4 * (int64_t)G * per;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n; e += stride) {
    const int co = (int)(e % Cout), t = (int)((e / Cout) % 9), ci = (int)((e / (9 * Cout)) % Cin);
    const int64_t gp = e / per;
    const int g = (int)(gp % G), ph = (int)(gp / G);
    const int dr = t / 3 - 1, dc = t % 3 - 1;
    const int kh = (ph >> 1) + 1 - 2 * dr, kw = (ph & 1) + 1 - 2 * dc;
    uint16_t v = 0;
    if (kh >= 0 && kh <= 2 && kw >= 0 && kw <= 2)
      v = Wb[(int64_t)g * d_pad + w_off + (((int64_t)co * 3 + kh) * 3 + kw) * Cin + ci];
    wt4[e] = v;
  }
}

// Every data gradient's flipped weights of a step in one launch (the weights do not change during
// the backward): job k covers elements [begin_k, begin_k + n_k) and writes what
// flip_weights_kernel (phases = 0) or flip_phase_weights_kernel (phases = 1) would, to dst_k.
struct FlipJob {
  int64_t w_off;   // the layer's weights within each replica's d_pad slice
  uint16_t* dst;   // [G][Cin][9][Cout], or [4][G][Cin][9][Cout] with phases
  int64_t begin;   // first element of this job
  int64_t n;       // its elements
  int cin, cout, phases, pad;
};
constexpr int kMaxFlipJobs = 24;
struct FlipJobs {
  int n;
  FlipJob j[kMaxFlipJobs];
};

__global__ void flip_jobs_kernel(const uint16_t* __restrict__ Wb, int64_t d_pad, int G,
                                 const __grid_constant__ FlipJobs js, int64_t total) {
  pdl_begin();
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total; t += stride) {
    int k = 0;
    while (k + 1 < js.n && t >= js.j[k + 1].begin) ++k;
    const FlipJob& jb = js.j[k];
    const int64_t e = t - jb.begin;
    const int Cin = jb.cin, Cout = jb.cout;
    const int64_t per = (int64_t)Cin * 9 * Cout;
    const int co = (int)(e % Cout), tp = (int)((e / Cout) % 9), ci = (int)((e / (9 * Cout)) % Cin);
    const int64_t gp = e / per;
    if (!jb.phases) {
      const int g = (int)gp;
      jb.dst[e] = Wb[(int64_t)g * d_pad + jb.w_off + ((int64_t)co * 9 + (8 - tp)) * Cin + ci];
    } else {
      const int g = (int)(gp % G), ph = (int)(gp / G);
      const int dr = tp / 3 - 1, dc = tp % 3 - 1;
      const int kh = (ph >> 1) + 1 - 2 * dr, kw = (ph & 1) + 1 - 2 * dc;
      uint16_t v = 0;
      if (kh >= 0 && kh <= 2 && kw >= 0 && kw <= 2)
        v = Wb[(int64_t)g * d_pad + jb.w_off + (((int64_t)co * 3 + kh) * 3 + kw) * Cin + ci];
      jb.dst[e] = v;
    }
  }
}

// The option-A shortcut's share of a block's input gradient: for input pixels on the stride grid
// and the first Cin channels, dx += dout * (out > 0) at (ih / s, iw / s).  Thread = (output pixel,
// 4 channels < Cin), blockIdx.y the replica; only the input pixels on the stride grid are touched.
template <typename TA>
__global__ void __launch_bounds__(256) add_shortcut_grad_v2_kernel(
    float* __restrict__ dx, const float* __restrict__ dout, const TA* __restrict__ out, int B,
    int Hin, int Win, int Cin, int Hout, int Wout, int Cout, int stride) {
  pdl_begin();
  const int g = blockIdx.y, C4 = Cin / 4;
  const int Po = B * Hout * Wout;
  const int e = blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= Po * C4) return;
  const int po = e / C4, c0 = (e - po * C4) * 4;
  const int64_t o = ((int64_t)g * Po + po) * Cout + c0;
  int64_t i;
  if (stride == 1 && Hin == Hout && Win == Wout) {
    i = ((int64_t)g * Po + po) * Cin + c0;  // identity shortcut: the same pixel
  } else {
    const int ow = po % Wout, t2 = po / Wout, oh = t2 % Hout, b = t2 / Hout;
    i = ((((int64_t)g * B + b) * Hin + oh * stride) * Win + ow * stride) * Cin + c0;
  }
  const float4 d = *reinterpret_cast<const float4*>(dout + o);
  const float4 a = Vec4<TA>::load(out + o);
  float4 x = *reinterpret_cast<float4*>(dx + i);
  x.x += a.x > 0.f ? d.x : 0.f;
  x.y += a.y > 0.f ? d.y : 0.f;
  x.z += a.z > 0.f ? d.z : 0.f;
  x.w += a.w > 0.f ? d.w : 0.f;
  *reinterpret_cast<float4*>(dx + i) = x;
}

}  // namespace

struct ResNetPlan {
  lsgd_config cfg{};
  int K = 0, B = 0, C = 0, H0 = 0, W0 = 0, C0 = 0, base = 0, blocks = 0, F = 0;
  bool bf16 = false;
  std::vector<ConvL> convs;
  int64_t fc_w = 0, fc_b = 0, c_fc_w = 0, c_fc_b = 0;
  int64_t d = 0, d_pad = 0, decay_end = 0;
  int64_t max_act = 0;  // largest activation tensor over all replicas (elements)
  void* x0 = nullptr;
  std::vector<void*> act;
  std::vector<float*> y, mean, rstd;
  float *feat = nullptr, *logits = nullptr, *dlogits = nullptr, *dfeat = nullptr;
  float* dA[2] = {nullptr, nullptr};
  float* dh = nullptr;
  void* dy = nullptr;
  float* part = nullptr;
  size_t part_floats = 0;
  float* s12 = nullptr;
  // weight-gradient partials of each tensor-core weight gradient (null where none), kept until
  // the end of the backward, whose one launch then sums all of them (sum_jobs: the pending sums)
  std::vector<float*> wpart;
  std::vector<SumJob> sum_jobs;
  // each data gradient's flipped weights (null where the step flips into the shared wt / wt4),
  // all written by one launch at the start of the backward
  std::vector<uint16_t*> wflip;
  // tensor-core convolutions (BF16 mode): per-convolution im2col of its input (kept from the
  // forward for the weight gradient), the output-gradient im2col and flipped weights of the
  // stride-1 data gradients
  bool tc = false;
  std::vector<uint16_t*> col;
  uint16_t* colT = nullptr;
  uint16_t* wt = nullptr;
  // a stem with fewer than 16 input channels runs as a 16-channel convolution on the tensor-core
  // kernels: the image with zero channels appended, and its weights likewise
  bool stem16 = false;
  uint16_t* x16 = nullptr;    // [K][B][H0][W0][16]
  uint16_t* wstem = nullptr;  // [K][Cout][9][16]
  // the stride-2 data gradients as four parity phases on the implicit kernel: their weights
  uint16_t* wt4 = nullptr;    // [4][K][Cin][9][Cout] of the largest such convolution
  // BatchNorm statistics computed by the forward convolutions' epilogues: per replica, CTA and
  // epilogue warp, (count, mean, M2) of each channel, merged by bn_merge_partials_kernel
  float4* cstats = nullptr;   // [K + 2 SMs][64]
  // backward BatchNorm sums computed by the data-gradient convolutions' epilogues (ConvBwdFuse),
  // consumed by the next BatchNorm backward: [K][16 (K + 2 SMs) / K][64] at most
  float2* bpart = nullptr;
  std::string err;
};

namespace {

// The weight-gradient kernel (partials into part) and their ordered sum into dW.  With defer, a
// sum that the 4-wide kernel takes is not launched but described in *defer (*deferred = true), to
// run with the step's others in one launch.
cudaError_t launch_conv_wgrad_impl(const uint16_t* x, const uint16_t* dy, float* dW, int64_t dW_gs,
                                   int G, int B, int hout, int wout, int cin, int cout, int stride,
                                   float* part, cudaStream_t s, int cin_out, SumJob* defer,
                                   bool* deferred) {
  if (deferred) *deferred = false;
  const int hin = hout * stride, win = wout * stride;
  const int64_t P = (int64_t)B * hout * wout;
  if (cin_out <= 0) cin_out = cin;
  if (!conv_wgrad_tc_ok(cin, cout, stride, hin, win, hout, wout) || G < 1 || B < 1 ||
      P > 0x7fffffffLL || cin_out > cin)
    return cudaErrorInvalidValue;
  ConvWgradArgs a{};
  // the output-gradient tile: 64 pixels x nb channels (Cout of 16 / 32 / 64 exactly; 48 padded
  // to 64 by the map's zero fill), swizzled at its 2 nb-byte row
  const int nb = (cout == 16 || cout == 32) ? cout : 64;
  if (!make_tma_map_halo(&a.x_map, x, cin, win, hin, B, G, stride, wout) ||
      !make_tma_map(&a.dy_map, dy, true, cout, P, G, cout, (uint64_t)P * cout, nb, 64, 2 * nb))
    return cudaErrorInvalidValue;
  a.nb = nb;
  a.cin = cin;
  a.cout = cout;
  a.stride = stride;
  a.hin = hin;
  a.win = win;
  a.hout = hout;
  a.wout = wout;
  a.G = G;
  a.P = (int)P;
  a.cpr = conv_wgrad_ctas(cin, stride, wout, G, P);
  a.part = part;
  cudaError_t e = launch_conv_wgrad_tc(a, s);
  if (e != cudaSuccess) return e;
  // the partials' sum, cropped to the first cin_out channels of every tap
  if (defer && deferred && sum_partials_v4_ok(part, 9 * cin, 9 * cin_out, dW, dW_gs, cin, cin_out)) {
    *defer = SumJob{part, dW, dW_gs, 0, a.cpr, cout, 9 * cin, 9 * cin_out, G, cin, cin_out, 0};
    *deferred = true;
    return cudaGetLastError();
  }
  launch_sum_partials(part, a.cpr, cout, 9 * cin, 9 * cin_out, G, dW, dW_gs, cin, cin_out, s);
  return cudaGetLastError();
}


size_t esz(const ResNetPlan* p) { return p->bf16 ? 2 : 4; }

lsgd_status rn_check(ResNetPlan* p, int64_t* launches, cudaError_t e, const char* what) {
  if (launches) ++*launches;
  if (e != cudaSuccess) {
    p->err = std::string(what) + ": " + cudaGetErrorString(e);
    return LSGD_ECUDA;
  }
  return LSGD_OK;
}

// A raw kernel launch (its error is the launch's last error) ...
#define RN_LAUNCH(expr)                                                              \
  do {                                                                               \
    expr;                                                                            \
    const lsgd_status st__ = rn_check(p, launches, cudaGetLastError(), #expr);       \
    if (st__ != LSGD_OK) return st__;                                                \
  } while (0)
// ... or a launcher returning a cudaError_t (which also reports rejected arguments).
#define RN_CALL(expr)                                                                \
  do {                                                                               \
    const lsgd_status st__ = rn_check(p, launches, (expr), #expr);                   \
    if (st__ != LSGD_OK) return st__;                                                \
  } while (0)

int64_t conv_pixels(const ResNetPlan* p, const ConvL& c) { return (int64_t)p->B * c.hout * c.wout; }

bool conv_on_tc(const ResNetPlan* p, const ConvL& c) { return p->tc && c.cout % 8 == 0; }
// Row length of a convolution's column matrix: 9 Cin rounded up to a multiple of 8 elements.
int col_ld(const ConvL& c) { return (int)rup(9 * c.cin, 8); }

int grid_for_items(int64_t n) { return grid_cap(n, 256); }
// Implicit-GEMM convolutions on the tensor cores: Ck = 16, 32 or 64 channels per tap, an output
// that tiles into 128-pixel blocks of whole rows (see conv_tile_shape), stride 1 or 2.
bool implicit_conv_ok(int ck, int stride, int hout, int wout) {
  int rows = 0, images = 0;
  return (ck == 16 || ck == 32 || ck == 64) && (stride == 1 || stride == 2) &&
         conv_tile_shape(hout, wout, &rows, &images);
}
// The weight gradient builds its column matrix in shared memory (conv_wgrad_tc_kernel).
bool wgrad_tc(const ResNetPlan* p, const ConvL& c) {
  return conv_on_tc(p, c) && conv_wgrad_tc_ok(c.cin, c.cout, c.stride, c.hin, c.win, c.hout, c.wout);
}
// The forward reads the input straight from the activation (implicit GEMM).
bool implicit_fwd(const ConvL& c) {
  return implicit_conv_ok(c.cin, c.stride, c.hout, c.wout) && col_ld(c) == 9 * c.cin;
}
// A tensor-core convolution whose forward or weight gradient needs the column matrix in HBM.
bool needs_col(const ResNetPlan* p, const ConvL& c) {
  return conv_on_tc(p, c) && !(wgrad_tc(p, c) && implicit_fwd(c));
}

// The persistent convolution kernel: N = 16, 32 or 64 outputs, whole 128-pixel tiles.
bool persistent_conv_ok(int n, int64_t P) { return (n == 16 || n == 32 || n == 64) && P % 128 == 0; }
// The stem (fewer than 16 input channels) as a 16-channel convolution on the implicit kernels.
bool stem16_ok(const ResNetPlan* p, const ConvL& c) {
  const int64_t P = (int64_t)p->B * c.hout * c.wout;
  return conv_on_tc(p, c) && c.cin < 16 && c.stride == 1 && implicit_conv_ok(16, 1, c.hout, c.wout) &&
         persistent_conv_ok(c.cout, P) &&
         conv_wgrad_tc_ok(16, c.cout, 1, c.hin, c.win, c.hout, c.wout);
}
// A stride-2 data gradient as four parity phases on the persistent implicit-GEMM kernel.
bool phase_dgrad_ok(const ResNetPlan* p, const ConvL& c) {
  return conv_on_tc(p, c) && c.stride == 2 && c.hin == 2 * c.hout && c.win == 2 * c.wout &&
         implicit_conv_ok(c.cout, 1, c.hout, c.wout) &&
         persistent_conv_ok(c.cin, (int64_t)p->B * c.hout * c.wout);
}
// The four-channel kernels need C a multiple of 4 with C / 4 dividing their 256 threads.
bool vec4_ok(int C) { return C % 4 == 0 && 256 % (C / 4) == 0; }
// Blocks of a per-replica kernel whose threads each take one pixel and group of 4 channels.
unsigned px_blocks(int64_t P, int C) {
  const int64_t ppb = 256 / (C / 4);
  return (unsigned)std::max<int64_t>(1, std::min<int64_t>((P + ppb - 1) / ppb, (int64_t)kNumSMs * 8));
}

// ---- 3x3 convolutions on the persistent implicit-GEMM kernel (conv_tc_kernel), raw pointers ----
// The ResNet-20 step and the stand-alone lsgd_conv3x3_bf16 entry point both run these, so the
// element-wise kernel tests cover the step's own launches.  Weights w [G][Cout][3][3][Cin] bf16
// with replica stride w_gs; activations NHWC bf16; outputs fp32, fully overwritten.

#define CV_LAUNCH(expr)                                                              \
  do {                                                                               \
    expr;                                                                            \
    if (launches) ++*launches;                                                       \
    const cudaError_t e__ = cudaGetLastError();                                      \
    if (e__ != cudaSuccess) {                                                        \
      err = std::string(#expr) + ": " + cudaGetErrorString(e__);                     \
      return LSGD_ECUDA;                                                             \
    }                                                                                \
  } while (0)
#define CV_CALL(expr)                                                                \
  do {                                                                               \
    if (launches) ++*launches;                                                       \
    const cudaError_t e__ = (expr);                                                  \
    if (e__ != cudaSuccess) {                                                        \
      err = std::string(#expr) + ": " + cudaGetErrorString(e__);                     \
      return LSGD_ECUDA;                                                             \
    }                                                                                \
  } while (0)

// Output size of a 3x3, padding-1 convolution.
int conv_out_size(int n, int stride) { return (n - 1) / stride + 1; }

// The forward y = conv(x, w) runs on the implicit kernel: the stem form (fewer than 16 input
// channels, padded to 16) or the direct form (16, 32 or 64 channels per tap).
bool conv_fwd_tc_route(int B, int hin, int win, int cin, int cout, int stride) {
  const int hout = conv_out_size(hin, stride), wout = conv_out_size(win, stride);
  const int64_t P = (int64_t)B * hout * wout;
  if (cout % 8 || P > 0x7fffffffLL) return false;
  if (cin < 16)
    return stride == 1 && implicit_conv_ok(16, 1, hout, wout) && persistent_conv_ok(cout, P);
  return implicit_conv_ok(cin, stride, hout, wout) && persistent_conv_ok(cout, P);
}

// The data gradient dx = conv^T(dy, w) runs on the implicit kernel: stride 1 as a convolution of
// dy with the flipped, transposed weights; stride 2 as four parity phases.
bool conv_dgrad_tc_route(int B, int hin, int win, int cin, int cout, int stride) {
  const int hout = conv_out_size(hin, stride), wout = conv_out_size(win, stride);
  if (cout % 8 || cin % 8 || (int64_t)B * hin * win > 0x7fffffffLL) return false;
  if (stride == 1) return implicit_conv_ok(cout, 1, hin, win) && persistent_conv_ok(cin, (int64_t)B * hin * win);
  return stride == 2 && hin == 2 * hout && win == 2 * wout && implicit_conv_ok(cout, 1, hout, wout) &&
         persistent_conv_ok(cin, (int64_t)B * hout * wout);
}

// Scratch of the forward's stem form (x16 [G][B][hin][win][16], wstem [G][cout][9][16]) and of
// the data gradient (stride 1: wt [G][cin][9][cout]; stride 2: wt4 [4][G][cin][9][cout]), bf16.
size_t conv_x16_elems(int G, int B, int hin, int win) { return (size_t)G * B * hin * win * 16; }
size_t conv_wstem_elems(int G, int cout) { return (size_t)G * cout * 9 * 16; }
size_t conv_wt_elems(int G, int cin, int cout, int stride) {
  return (size_t)(stride == 2 ? 4 : 1) * G * cin * 9 * cout;
}

lsgd_status conv_fwd_tc(const uint16_t* x, const uint16_t* w, int64_t w_gs, float* y, int G, int B,
                        int hin, int win, int cin, int cout, int stride, uint16_t* x16,
                        uint16_t* wstem, cudaStream_t s, std::string& err, int64_t* launches,
                        float4* stats = nullptr, int* nparts = nullptr) {
  if (!conv_fwd_tc_route(B, hin, win, cin, cout, stride)) {
    err = "convolution shape not taken by the implicit-GEMM kernel";
    return LSGD_EUNSUPPORTED;
  }
  const int hout = conv_out_size(hin, stride), wout = conv_out_size(win, stride);
  const int64_t P = (int64_t)B * hout * wout;
  ConvArgs ca{};
  bool okc;
  if (cin < 16) {
    // the stem: zero channels appended to the image and the weights (the products are unchanged)
    const int64_t npix = (int64_t)G * B * hin * win;
    CV_LAUNCH(launch_pdl(pad_input16_kernel, grid_cap(npix, 256), 256, 0, s, x, x16, npix, cin));
    CV_LAUNCH(launch_pdl(pad_stem_weights_kernel, grid_cap((int64_t)G * cout * 144, 256), 256, 0, s,
                         w, w_gs, (int64_t)0, wstem, G, cout, cin));
    ca.strip = conv_strip_ok(hout, wout, 1);
    okc = make_tma_map_conv(&ca.in_map, x16, 16, win, hin, B, G, wout, hout, 1, ca.strip);
    okc &= make_tma_map(&ca.w_map, wstem, true, 9 * 16, cout, G, 9 * 16, (uint64_t)cout * 9 * 16, 16,
                        cout, 32);
    ca.ck = 16;
  } else {
    ca.strip = conv_strip_ok(hout, wout, stride);
    okc = make_tma_map_conv(&ca.in_map, x, cin, win, hin, B, G, wout, hout, stride, ca.strip);
    okc &= make_tma_map(&ca.w_map, w, true, 9 * cin, cout, G, 9 * cin, w_gs, cin, cout, 2 * cin);
    ca.ck = cin;
  }
  if (!okc) {
    err = "TMA map encoding failed (implicit convolution)";
    return LSGD_ECUDA;
  }
  ca.stride = cin < 16 ? 1 : stride;
  ca.hout = hout;
  ca.wout = wout;
  ca.N = ca.np = cout;
  ca.G = G;
  ca.P = (int)P;
  ca.out = y;
  ca.out_gs = P * cout;
  ca.stats = stats;
  CV_CALL(launch_conv_tc(ca, s, stats ? nparts : nullptr));
  return LSGD_OK;
}

// bf (optional): the BatchNorm-backward epilogue (ConvBwdFuse; part_gs / part_off are filled in
// here); *nparts receives the partials per replica it wrote.
// flipped: wt already holds the flipped (stride 2: the four phases') weights of w.
lsgd_status conv_dgrad_tc(const uint16_t* dy, const uint16_t* w, int64_t w_gs, float* dx, int G,
                          int B, int hin, int win, int cin, int cout, int stride, uint16_t* wt,
                          cudaStream_t s, std::string& err, int64_t* launches,
                          const ConvBwdFuse* bf = nullptr, int* nparts = nullptr,
                          bool flipped = false) {
  if (nparts) *nparts = 0;
  if (!conv_dgrad_tc_route(B, hin, win, cin, cout, stride)) {
    err = "data-gradient shape not taken by the implicit-GEMM kernel";
    return LSGD_EUNSUPPORTED;
  }
  const int64_t P = (int64_t)B * hin * win;
  if (stride == 1) {
    if (!flipped)
      CV_LAUNCH((launch_pdl(flip_weights_kernel, dim3((unsigned)((cin * 9 * cout + 255) / 256), (unsigned)G),
                            256, 0, s, w, w_gs, (int64_t)0, wt, G, cin, cout)));
    ConvArgs ca{};
    ca.strip = conv_strip_ok(hin, win, 1);
    bool okc = make_tma_map_conv(&ca.in_map, dy, cout, win, hin, B, G, win, hin, 1, ca.strip);
    okc &= make_tma_map(&ca.w_map, wt, true, 9 * cout, cin, G, 9 * cout, (uint64_t)cin * 9 * cout,
                        cout, cin, 2 * cout);
    if (!okc) {
      err = "TMA map encoding failed (implicit data gradient)";
      return LSGD_ECUDA;
    }
    ca.ck = cout;
    ca.stride = 1;
    ca.hout = hin;
    ca.wout = win;
    ca.N = ca.np = cin;
    ca.G = G;
    ca.P = (int)P;
    ca.out = dx;
    ca.out_gs = P * cin;
    if (bf) {
      ca.bwd = *bf;
      const int cpr = conv_tc_ctas(ca);
      if (cpr < 1) {
        err = "data-gradient arguments rejected";
        return LSGD_EINVAL;
      }
      ca.bwd.part_gs = 4 * cpr;
      ca.bwd.part_off = 0;
      if (nparts) *nparts = 4 * cpr;
    }
    CV_CALL(launch_conv_tc(ca, s));
    return LSGD_OK;
  }
  // stride 2: each parity phase of dx is a 3x3 stride-1 convolution of dy (weights of the phase's
  // taps, zeros elsewhere) whose outputs land on every other row and column of dx
  const int hout = hin / 2, wout = win / 2;
  const int64_t per = (int64_t)cin * 9 * cout;
  if (!flipped)
    CV_LAUNCH(launch_pdl(flip_phase_weights_kernel, grid_cap(4 * (int64_t)G * per, 256), 256, 0, s,
                         w, w_gs, (int64_t)0, wt, G, cin, cout));
  const int64_t Pq = (int64_t)B * hout * wout;
  for (int ph = 0; ph < 4; ++ph) {
    ConvArgs ca{};
    ca.strip = conv_strip_ok(hout, wout, 1);
    bool okc = make_tma_map_conv(&ca.in_map, dy, cout, wout, hout, B, G, wout, hout, 1, ca.strip);
    okc &= make_tma_map(&ca.w_map, wt + ph * G * per, true, 9 * cout, cin, G, 9 * cout,
                        (uint64_t)per, cout, cin, 2 * cout);
    if (!okc) {
      err = "TMA map encoding failed (stride-2 data gradient)";
      return LSGD_ECUDA;
    }
    ca.ck = cout;
    ca.stride = 1;
    ca.hout = hout;
    ca.wout = wout;
    ca.N = ca.np = cin;
    ca.G = G;
    ca.P = (int)Pq;
    ca.out = dx;
    ca.out_gs = P * cin;
    ca.ph_y = ph >> 1;
    ca.ph_x = ph & 1;
    ca.dst_h = hin;
    ca.dst_w = win;
    if (bf) {
      // the four phases' partials side by side: phase ph writes partials [4 cpr ph, 4 cpr (ph + 1))
      ca.bwd = *bf;
      const int cpr = conv_tc_ctas(ca);
      if (cpr < 1) {
        err = "data-gradient arguments rejected";
        return LSGD_EINVAL;
      }
      ca.bwd.part_gs = 16 * cpr;
      ca.bwd.part_off = 4 * cpr * ph;
      if (nparts) *nparts = 16 * cpr;
    }
    CV_CALL(launch_conv_tc(ca, s));
  }
  return LSGD_OK;
}

// stats / nparts: where the persistent implicit kernel runs, it also writes the output's
// partial BatchNorm statistics to stats and their count per replica to *nparts (else 0).
template <typename TA>
lsgd_status conv_forward(ResNetPlan* p, int i, const void* in, const void* Wop, int w_g0,
                         int w_gmul, float* y, int G, cudaStream_t s, int64_t* launches,
                         float4* stats, int* nparts) {
  const ConvL& c = p->convs[i];
  const int64_t P = conv_pixels(p, c);
  *nparts = 0;
  if (i == 0 && p->stem16 && w_g0 == 0 && w_gmul == 1) {
    // the stem as a 16-channel convolution on the persistent implicit-GEMM kernel
    const lsgd_status st = conv_fwd_tc(reinterpret_cast<const uint16_t*>(in),
                                       reinterpret_cast<const uint16_t*>(Wop) + c.w_off, p->d_pad, y,
                                       G, p->B, c.hin, c.win, c.cin, c.cout, 1, p->x16, p->wstem, s,
                                       p->err, launches, stats, nparts);
    return st;
  }
  if (conv_on_tc(p, c) && w_g0 == 0 && w_gmul == 1) {
    // y = im2col(in) [P][9 Cin] x W^T on the tensor cores (both operands K-major)
    const int Kc = col_ld(c);
    const uint16_t* wop = reinterpret_cast<const uint16_t*>(Wop) + c.w_off;
    int64_t w_gs = p->d_pad;
    if (Kc == 9 * c.cin && !needs_col(p, c)) {
      // neither product needs the column matrix
    } else if (Kc == 9 * c.cin) {
      const uint16_t* in16 = reinterpret_cast<const uint16_t*>(in);
      const dim3 rows_grid((unsigned)(p->B * c.hout), (unsigned)G);
      if (c.cin == 16)
        RN_LAUNCH((launch_pdl(im2col_row_kernel<2>, rows_grid, 256, 0, s, in16, p->col[i], p->B,
            c.hin, c.win, c.hout, c.wout, c.stride)));
      else if (c.cin == 32)
        RN_LAUNCH((launch_pdl(im2col_row_kernel<4>, rows_grid, 256, 0, s, in16, p->col[i], p->B,
            c.hin, c.win, c.hout, c.wout, c.stride)));
      else if (c.cin == 64)
        RN_LAUNCH((launch_pdl(im2col_row_kernel<8>, rows_grid, 256, 0, s, in16, p->col[i], p->B,
            c.hin, c.win, c.hout, c.wout, c.stride)));
      else
        RN_LAUNCH((launch_pdl(im2col_v2_kernel,
            dim3((unsigned)((P * 9 * (c.cin / 8) + 255) / 256), (unsigned)G), 256, 0, s, in16,
            p->col[i], p->B, c.hin, c.win, c.cin, c.hout, c.wout, c.stride)));
    } else {
      RN_LAUNCH((launch_pdl(im2col_any_row_kernel<uint16_t>,
          dim3((unsigned)(p->B * c.hout), (unsigned)G), 256, 0, s,
          reinterpret_cast<const uint16_t*>(in), p->col[i], p->B, c.hin, c.win, c.cin, c.hout,
          c.wout, c.stride, Kc)));
      RN_LAUNCH((launch_pdl(pad_weights_kernel, grid_for_items((int64_t)G * c.cout * Kc), 256, 0, s,
          reinterpret_cast<const uint16_t*>(Wop), p->d_pad, c.w_off, p->wt, G, c.cout, 9 * c.cin,
          Kc)));
      wop = p->wt;
      w_gs = (int64_t)c.cout * Kc;
    }
    TcGemmArgs t{};
    t.M = (int)P;
    t.N = c.cout;
    t.Kd = Kc;
    t.G = G;
    if (implicit_conv_ok(c.cin, c.stride, c.hout, c.wout) && Kc == 9 * c.cin &&
        persistent_conv_ok(c.cout, P)) {
      // persistent implicit GEMM: the input tile of each tap straight from the NHWC activation
      // by TMA
      return conv_fwd_tc(reinterpret_cast<const uint16_t*>(in), wop, w_gs, y, G, p->B, c.hin, c.win,
                         c.cin, c.cout, c.stride, nullptr, nullptr, s, p->err, launches, stats,
                         nparts);
    }
    if (implicit_conv_ok(c.cin, c.stride, c.hout, c.wout) && Kc == 9 * c.cin) {
      // implicit GEMM: the input tile of each tap straight from the NHWC activation by TMA
      t.conv = 1;
      t.cv_ck = c.cin;
      t.cv_stride = c.stride;
      t.cv_hout = c.hout;
      t.cv_wout = c.wout;
      bool okc = make_tma_map_conv(&t.A.map, in, c.cin, c.win, c.hin, p->B, G, c.wout, c.hout,
                                   c.stride);
      okc &= make_tma_map(&t.B.map, wop, true, 9 * c.cin, c.cout, G, 9 * c.cin, w_gs, c.cin, 64,
                          2 * c.cin);
      if (!okc) {
        p->err = "TMA map encoding failed (implicit convolution)";
        return LSGD_ECUDA;
      }
      t.A.box_rows = kTcTileM;
      t.B.box_rows = 64;
      t.C = y;
      t.c_rs = c.cout;
      t.c_gs = P * c.cout;
      t.epi = EPI_STORE;
      RN_CALL(launch_gemm_tc(t, s));
      return LSGD_OK;
    }
    const int bn = tc_tile_n(Kc);
    bool ok = make_tma_map_bf16(&t.A.map, p->col[i], Kc, P, G, Kc, (uint64_t)P * Kc, 64, kTcTileM);
    ok &= make_tma_map_bf16(&t.B.map, wop, Kc, c.cout, G, Kc, w_gs, 64, bn);
    if (!ok) {
      p->err = "TMA map encoding failed (convolution)";
      return LSGD_ECUDA;
    }
    t.A.box_rows = kTcTileM;
    t.B.box_rows = bn;
    t.C = y;
    t.c_rs = c.cout;
    t.c_gs = P * c.cout;
    t.epi = EPI_STORE;
    RN_CALL(launch_gemm_tc(t, s));
    return LSGD_OK;
  }
  dim3 grid((unsigned)((P + 127) / 128), (unsigned)((c.cout + 15) / 16), (unsigned)G);
  const size_t smem = (size_t)16 * 9 * c.cin * 4;
  const TA* wbase = reinterpret_cast<const TA*>(Wop) + (int64_t)w_g0 * p->d_pad + c.w_off;
  RN_LAUNCH((launch_pdl(conv_fwd_kernel<TA>, grid, 128, smem, s, reinterpret_cast<const TA*>(in),
      wbase, (int64_t)w_gmul * p->d_pad, y, p->B, c.hin, c.win, c.cin, c.hout, c.wout, c.cout,
      c.stride)));
  return LSGD_OK;
}

lsgd_status bn_stats(ResNetPlan* p, const ConvL& c, const float* y, float* mean, float* rstd, int G,
                     cudaStream_t s, int64_t* launches) {
  const int64_t P = conv_pixels(p, c);
  const int chunk = rn_chunk(P);
  const int nq = (int)((P + chunk - 1) / chunk);
  const int lanes = std::max(1, 256 / c.cout);
  dim3 grid(nq, G);
  if (vec4_ok(c.cout))
    RN_LAUNCH((launch_pdl(bn_stats_partial_v4_kernel, grid, 256, 0, s, y, P, c.cout, nq, chunk,
        p->part)));
  else
    RN_LAUNCH((launch_pdl(bn_stats_partial_kernel, grid, lanes * c.cout, 0, s, y, P, c.cout, nq,
        chunk, p->part)));
  RN_LAUNCH((launch_pdl(bn_stats_finalize_kernel, (G * c.cout * 32 + 127) / 128, 128, 0, s, p->part,
      P, c.cout, nq, chunk, G, mean, rstd)));
  return LSGD_OK;
}

template <typename TA>
lsgd_status forward_impl(ResNetPlan* p, const float* W, const void* Wop, int w_g0, int w_gmul,
                         int G, cudaStream_t s, int64_t* launches) {
  const size_t n_conv = p->convs.size();
  for (size_t i = 0; i < n_conv; ++i) {
    const ConvL& c = p->convs[i];
    // block j uses convolutions 2j+1 (input act[2j], the block input) and 2j+2 (input act[2j+1])
    const void* in = i == 0 ? p->x0 : p->act[i - 1];
    // the convolution's epilogue forms the BatchNorm statistics where it can (one small kernel
    // merges its partials), else the two statistics passes run
    int nparts = 0;
    float4* cst = p->cstats && vec4_ok(c.cout) && c.cout <= 64 ? p->cstats : nullptr;
    lsgd_status st = conv_forward<TA>(p, (int)i, in, Wop, w_g0, w_gmul, p->y[i], G, s, launches,
                                      cst, &nparts);
    if (st != LSGD_OK) return st;
    if (nparts == 0) {
      st = bn_stats(p, c, p->y[i], p->mean[i], p->rstd[i], G, s, launches);
      if (st != LSGD_OK) return st;
    } else {
      RN_LAUNCH((launch_pdl(bn_merge_partials_kernel, (G * c.cout * 32 + 127) / 128, 128, 0, s,
          cst, nparts, G, c.cout, p->mean[i], p->rstd[i])));
    }
    const bool second = i > 0 && i % 2 == 0;
    const TA* sc = second ? reinterpret_cast<const TA*>(p->act[i - 2]) : nullptr;
    const ConvL& ca = p->convs[second ? i - 1 : i];
    if (vec4_ok(c.cout)) {
      RN_LAUNCH((launch_pdl(bn_act_fwd_v4_kernel<TA>,
          dim3(px_blocks(conv_pixels(p, c), c.cout), (unsigned)G), 256, 0, s, p->y[i], p->mean[i],
          p->rstd[i], W, c.g_off, c.b_off, p->d_pad, w_g0, w_gmul, sc, ca.hin, ca.win, ca.cin,
          ca.stride, reinterpret_cast<TA*>(p->act[i]), p->B, c.hout, c.wout, c.cout)));
    } else {
      const int64_t n = (int64_t)G * conv_pixels(p, c) * c.cout / 4;
      RN_LAUNCH((launch_pdl(bn_act_fwd_kernel<TA>, grid_cap(n, 256), 256, 0, s, p->y[i], p->mean[i],
          p->rstd[i], W, c.g_off, c.b_off, p->d_pad, w_g0, w_gmul, sc, ca.hin, ca.win, ca.cin,
          ca.stride, reinterpret_cast<TA*>(p->act[i]), G, p->B, c.hout, c.wout, c.cout)));
    }
  }
  // global average pooling and the classifier (fp32)
  const ConvL& last = p->convs.back();
  const int HW = last.hout * last.wout;
  RN_LAUNCH((launch_pdl(avgpool_kernel<TA>, (G * p->B * p->F + 127) / 128, 128, 0, s,
      reinterpret_cast<const TA*>(p->act.back()), p->feat, G * p->B, HW, p->F)));
  GemmArgs g{};
  g.M = p->B;
  g.N = p->C;
  g.Kd = p->F;
  g.G = G;
  g.A = p->feat;
  g.a_rs = p->F;
  g.a_cs = 1;
  g.a_gs = (int64_t)p->B * p->F;
  g.B = W + (int64_t)w_g0 * p->d_pad + p->fc_w;
  g.b_rs = 1;
  g.b_cs = p->F;
  g.b_gs = (int64_t)w_gmul * p->d_pad;
  g.C = p->logits;
  g.c_rs = p->C;
  g.c_gs = (int64_t)p->B * p->C;
  g.epi = EPI_BIAS;
  g.bias = W + (int64_t)w_g0 * p->d_pad + p->fc_b;
  g.bias_gs = (int64_t)w_gmul * p->d_pad;
  RN_CALL(launch_gemm_simt(g, s));
  return LSGD_OK;
}

// fused_parts > 0: the data-gradient convolution that produced dout already masked it by out > 0
// and left the sums' partials in p->bpart (ConvBwdFuse); only their merge and the apply pass run.
template <typename TA>
lsgd_status bn_backward(ResNetPlan* p, const ConvL& c, int i, const float* dout, const void* out,
                        const float* W, float* Gr, cudaStream_t s, int64_t* launches,
                        int fused_parts = 0) {
  const int K = p->K;
  const int64_t P = conv_pixels(p, c);
  const int chunk = rn_chunk(P);
  const int nq = (int)((P + chunk - 1) / chunk);
  const int lanes = std::max(1, 256 / c.cout);
  if (fused_parts > 0) {
    RN_LAUNCH((launch_pdl(bn_bwd_merge_kernel, (K * c.cout * 32 + 127) / 128, 128, 0, s, p->bpart,
        fused_parts, c.cout, K, p->s12, Gr, c.g_off, c.b_off, p->d_pad)));
  } else if (vec4_ok(c.cout))
    RN_LAUNCH((launch_pdl(bn_bwd_partial_v4_kernel<TA>, dim3(nq, K), 256, 0, s, dout,
        reinterpret_cast<const TA*>(out), p->y[i], p->mean[i], p->rstd[i], P, c.cout, nq, chunk,
        p->part)));
  else
    RN_LAUNCH((launch_pdl(bn_bwd_partial_kernel<TA>, dim3(nq, K), lanes * c.cout, 0, s, dout,
        reinterpret_cast<const TA*>(out), p->y[i], p->mean[i], p->rstd[i], P, c.cout, nq, chunk,
        p->part)));
  if (fused_parts == 0)
    RN_LAUNCH((launch_pdl(bn_bwd_finalize_kernel, (K * c.cout * 32 + 127) / 128, 128, 0, s,
        p->part, c.cout, nq, K, p->s12, Gr, c.g_off, c.b_off, p->d_pad)));
  if (vec4_ok(c.cout)) {
    // with fused partials dout is already masked: no read of the activation for the mask
    RN_LAUNCH((launch_pdl(bn_bwd_apply_v4_kernel<TA>, dim3(px_blocks(P, c.cout), (unsigned)K), 256,
        0, s, dout, fused_parts > 0 ? nullptr : reinterpret_cast<const TA*>(out), p->y[i],
        p->mean[i], p->rstd[i], p->s12, W, c.g_off, p->d_pad, reinterpret_cast<TA*>(p->dy),
        (int)P, c.cout)));
  } else {
    const int64_t n = (int64_t)K * P * c.cout / 4;
    RN_LAUNCH((launch_pdl(bn_bwd_apply_kernel<TA>, grid_cap(n, 256), 256, 0, s, dout,
        reinterpret_cast<const TA*>(out), p->y[i], p->mean[i], p->rstd[i], p->s12, W, c.g_off,
        p->d_pad, reinterpret_cast<TA*>(p->dy), K, P, c.cout)));
  }
  return LSGD_OK;
}

template <typename TA>
lsgd_status conv_wgrad(ResNetPlan* p, int i, const void* in, float* Gr, cudaStream_t s,
                       int64_t* launches) {
  const ConvL& c = p->convs[i];
  const int K = p->K;
  const int64_t P = conv_pixels(p, c);
  if (i == 0 && p->stem16) {
    // the padded stem's input (written by the forward); the gradient keeps the real channels
    RN_CALL(launch_conv_wgrad_bf16(p->x16, reinterpret_cast<const uint16_t*>(p->dy), Gr + c.w_off,
                                   p->d_pad, K, p->B, c.hout, c.wout, 16, c.cout, 1, p->part, s,
                                   c.cin));
    ++*launches;  // the partials' sum
    return LSGD_OK;
  }
  if (wgrad_tc(p, c)) {
    // dW [Cout][9 Cin] from dy and the input directly: the column matrix of each 64-pixel block
    // is built in shared memory; one partial per CTA, summed in order
    // with a buffer of its own the partials' sum waits for the end of the backward, where one
    // launch adds every layer's
    float* wp = (size_t)i < p->wpart.size() ? p->wpart[i] : nullptr;
    SumJob job{};
    bool deferred = false;
    const bool can_defer = wp && p->sum_jobs.size() < (size_t)kMaxSumJobs;
    RN_CALL(launch_conv_wgrad_impl(reinterpret_cast<const uint16_t*>(in),
                                   reinterpret_cast<const uint16_t*>(p->dy), Gr + c.w_off, p->d_pad,
                                   K, p->B, c.hout, c.wout, c.cin, c.cout, c.stride,
                                   wp ? wp : p->part, s, 0, can_defer ? &job : nullptr, &deferred));
    if (deferred)
      p->sum_jobs.push_back(job);
    else
      ++*launches;  // the partials' sum
    return LSGD_OK;
  }
  if (conv_on_tc(p, c)) {
    // dW [Cout][9 Cin] = dy^T [Cout][P] x im2col(in) [P][9 Cin]: both operands pixel-major
    // ("MN-major"); the pixel reduction is split across CTAs and the partials summed in order.
    const int Kc = col_ld(c);
    const int tiles = ((Kc + 63) / 64) * K;
    const int splits = tc_valid_splits((int)P, std::max(1, (4 * kNumSMs + tiles - 1) / tiles));
    TcGemmArgs t{};
    t.M = c.cout;
    t.N = Kc;
    t.Kd = (int)P;
    t.G = K;
    bool ok = make_tma_map_bf16(&t.A.map, p->dy, c.cout, P, K, c.cout, (uint64_t)P * c.cout, 64, 64);
    ok &= make_tma_map_bf16(&t.B.map, p->col[i], Kc, P, K, Kc, (uint64_t)P * Kc, 64, 64);
    if (!ok) {
      p->err = "TMA map encoding failed (convolution weight gradient)";
      return LSGD_ECUDA;
    }
    t.A.mn_major = t.B.mn_major = true;
    t.A.box_rows = t.B.box_rows = 64;
    t.C = p->part;
    t.c_rs = Kc;
    t.c_split_stride = (int64_t)c.cout * Kc;
    t.c_gs = (int64_t)splits * c.cout * Kc;
    t.splits = splits;
    t.epi = EPI_STORE;
    RN_CALL(launch_gemm_tc(t, s));
    RN_LAUNCH((launch_sum_partials(p->part, splits, c.cout, Kc, 9 * c.cin, K, Gr + c.w_off,
        p->d_pad, 0, 0, s)));
    return LSGD_OK;
  }
  const int nq = (int)((P + kWgradChunk - 1) / kWgradChunk);
  const int J = 9 * c.cin;
  const size_t smem = (size_t)(kWgradTile * 16 + kWgradTile * J) * 4;
  RN_LAUNCH((launch_pdl(conv_wgrad_partial_kernel<TA>, dim3(nq, (c.cout + 15) / 16, K), 256, smem,
      s, reinterpret_cast<const TA*>(p->dy), reinterpret_cast<const TA*>(in), p->part, p->B, c.hin,
      c.win, c.cin, c.hout, c.wout, c.cout, c.stride, nq)));
  const int64_t n = (int64_t)c.cout * J;
  RN_LAUNCH((launch_pdl(sum_partials_kernel, grid_cap((int64_t)K * n, 256), 256, 0, s, p->part, nq,
      n, K, Gr + c.w_off, p->d_pad)));
  return LSGD_OK;
}

// bn_t >= 0: convolution bn_t (whose output, the activation this data gradient flows into, is
// normalised next in the backward pass) gets its ReLU mask and BatchNorm-backward sums formed in
// the persistent kernel's epilogue, together with the shortcut's share of dout (ConvBwdFuse):
// dx then holds the masked gradient and *fused_parts the partials per replica in p->bpart (0 when
// this path did not run).
template <typename TA>
lsgd_status conv_dgrad(ResNetPlan* p, int i, const void* Wop, float* dx, const float* dout,
                       const void* out_act, cudaStream_t s, int64_t* launches, int bn_t = -1,
                       int* fused_parts = nullptr) {
  const ConvL& c = p->convs[i];
  const int K = p->K;
  const int64_t P = (int64_t)p->B * c.hin * c.win;
  if (fused_parts) *fused_parts = 0;
  ConvBwdFuse bf{};
  // measured per layer in the ResNet-20 step: the fused epilogue's extra loads pay for themselves
  // on the 16-channel data gradients (the largest tensors) but not on the 32 / 64-channel ones,
  // where the separate passes are cheaper than the epilogue's added latency
  const bool fuse = bn_t >= 0 && fused_parts && p->bpart && sizeof(TA) == 2 && c.cin <= 16;
  if (fuse) {
    bf.mask = reinterpret_cast<const uint16_t*>(p->act[bn_t]);
    bf.y = p->y[bn_t];
    bf.mean = p->mean[bn_t];
    bf.rstd = p->rstd[bn_t];
    if (dout) {
      bf.sc_dout = dout;
      bf.sc_out = reinterpret_cast<const uint16_t*>(out_act);
      bf.sc_C = c.cout;
      bf.sc_stride = c.stride;
      bf.sc_gs = (int64_t)p->B * c.hout * c.wout * c.cout;
    }
    bf.part = p->bpart;
  }
  if (conv_on_tc(p, c) && c.stride == 1 && implicit_conv_ok(c.cout, 1, c.hin, c.win)) {
    // stride 1: dx is the convolution of dy with the flipped, transposed weights -- an implicit
    // GEMM over dy's taps, no column matrix
    if (persistent_conv_ok(c.cin, P)) {
      uint16_t* wf = (size_t)i < p->wflip.size() ? p->wflip[i] : nullptr;
      const lsgd_status st = conv_dgrad_tc(reinterpret_cast<const uint16_t*>(p->dy),
                                           reinterpret_cast<const uint16_t*>(Wop) + c.w_off, p->d_pad,
                                           dx, K, p->B, c.hin, c.win, c.cin, c.cout, 1,
                                           wf ? wf : p->wt, s, p->err, launches,
                                           fuse ? &bf : nullptr, fused_parts, wf != nullptr);
      if (st != LSGD_OK) return st;
      if (fuse) return LSGD_OK;  // the epilogue added the shortcut's share
    } else {
      RN_LAUNCH((launch_pdl(flip_weights_kernel,
          dim3((unsigned)((c.cin * 9 * c.cout + 255) / 256), (unsigned)K), 256, 0, s,
          reinterpret_cast<const uint16_t*>(Wop), p->d_pad, c.w_off, p->wt, K, c.cin, c.cout)));
      TcGemmArgs t{};
      t.M = (int)P;
      t.N = c.cin;
      t.Kd = 9 * c.cout;
      t.G = K;
      t.conv = 1;
      t.cv_ck = c.cout;
      t.cv_stride = 1;
      t.cv_hout = c.hin;
      t.cv_wout = c.win;
      bool ok = make_tma_map_conv(&t.A.map, p->dy, c.cout, c.wout, c.hout, p->B, K, c.win, c.hin, 1);
      ok &= make_tma_map(&t.B.map, p->wt, true, 9 * c.cout, c.cin, K, 9 * c.cout,
                         (uint64_t)c.cin * 9 * c.cout, c.cout, 64, 2 * c.cout);
      if (!ok) {
        p->err = "TMA map encoding failed (implicit data gradient)";
        return LSGD_ECUDA;
      }
      t.A.box_rows = kTcTileM;
      t.B.box_rows = 64;
      t.C = dx;
      t.c_rs = c.cin;
      t.c_gs = P * c.cin;
      t.epi = EPI_STORE;
      RN_CALL(launch_gemm_tc(t, s));
    }
    if (dout) {
      const int64_t n = (int64_t)p->B * c.hout * c.wout * (c.cin / 4);
      RN_LAUNCH((launch_pdl(add_shortcut_grad_v2_kernel<TA>,
          dim3((unsigned)((n + 255) / 256), (unsigned)K), 256, 0, s, dx, dout,
          reinterpret_cast<const TA*>(out_act), p->B, c.hin, c.win, c.cin, c.hout, c.wout, c.cout,
          c.stride)));
    }
    return LSGD_OK;
  }
  if (phase_dgrad_ok(p, c)) {
    // stride 2: four parity phases on the persistent implicit-GEMM kernel
    uint16_t* wf = (size_t)i < p->wflip.size() ? p->wflip[i] : nullptr;
    const lsgd_status st = conv_dgrad_tc(reinterpret_cast<const uint16_t*>(p->dy),
                                         reinterpret_cast<const uint16_t*>(Wop) + c.w_off, p->d_pad,
                                         dx, K, p->B, c.hin, c.win, c.cin, c.cout, 2,
                                         wf ? wf : p->wt4, s, p->err, launches,
                                         fuse ? &bf : nullptr, fused_parts, wf != nullptr);
    if (st != LSGD_OK) return st;
    if (fuse) return LSGD_OK;  // the epilogue added the shortcut's share
    if (dout) {
      const int64_t n = (int64_t)p->B * c.hout * c.wout * (c.cin / 4);
      RN_LAUNCH((launch_pdl(add_shortcut_grad_v2_kernel<TA>,
          dim3((unsigned)((n + 255) / 256), (unsigned)K), 256, 0, s, dx, dout,
          reinterpret_cast<const TA*>(out_act), p->B, c.hin, c.win, c.cin, c.hout, c.wout, c.cout,
          c.stride)));
    }
    return LSGD_OK;
  }
  if (conv_on_tc(p, c) && c.cin % 8 == 0) {
    // dx = col(dy) [P][9 Cout] x wt^T with the flipped, transposed weights (stride 1 or 2)
    const int Kc = 9 * c.cout;
    const dim3 rows_grid((unsigned)(p->B * c.hin), (unsigned)K);
    const uint16_t* dy16 = reinterpret_cast<const uint16_t*>(p->dy);
    if (c.cout == 16)
      RN_LAUNCH((launch_pdl(col_dgrad_row_kernel<2>, rows_grid, 256, 0, s, dy16, p->colT, p->B,
          c.hin, c.win, c.hout, c.wout, c.stride)));
    else if (c.cout == 32)
      RN_LAUNCH((launch_pdl(col_dgrad_row_kernel<4>, rows_grid, 256, 0, s, dy16, p->colT, p->B,
          c.hin, c.win, c.hout, c.wout, c.stride)));
    else if (c.cout == 64)
      RN_LAUNCH((launch_pdl(col_dgrad_row_kernel<8>, rows_grid, 256, 0, s, dy16, p->colT, p->B,
          c.hin, c.win, c.hout, c.wout, c.stride)));
    else
      RN_LAUNCH((launch_pdl(col_dgrad_v2_kernel,
          dim3((unsigned)((P * 9 * (c.cout / 8) + 255) / 256), (unsigned)K), 256, 0, s,
          reinterpret_cast<const uint16_t*>(p->dy), p->colT, p->B, c.hin, c.win, c.cout, c.hout,
          c.wout, c.stride)));
    RN_LAUNCH((launch_pdl(flip_weights_kernel,
        dim3((unsigned)((c.cin * Kc + 255) / 256), (unsigned)K), 256, 0, s,
        reinterpret_cast<const uint16_t*>(Wop), p->d_pad, c.w_off, p->wt, K, c.cin, c.cout)));
    TcGemmArgs t{};
    t.M = (int)P;
    t.N = c.cin;
    t.Kd = Kc;
    t.G = K;
    const int bn = tc_tile_n(Kc);
    bool ok = make_tma_map_bf16(&t.A.map, p->colT, Kc, P, K, Kc, (uint64_t)P * Kc, 64, kTcTileM);
    ok &= make_tma_map_bf16(&t.B.map, p->wt, Kc, c.cin, K, Kc, (uint64_t)c.cin * Kc, 64, bn);
    if (!ok) {
      p->err = "TMA map encoding failed (convolution data gradient)";
      return LSGD_ECUDA;
    }
    t.A.box_rows = kTcTileM;
    t.B.box_rows = bn;
    t.C = dx;
    t.c_rs = c.cin;
    t.c_gs = P * c.cin;
    t.epi = EPI_STORE;
    RN_CALL(launch_gemm_tc(t, s));
    if (dout) {
      const int64_t n = (int64_t)p->B * c.hout * c.wout * (c.cin / 4);
      RN_LAUNCH((launch_pdl(add_shortcut_grad_v2_kernel<TA>,
          dim3((unsigned)((n + 255) / 256), (unsigned)K), 256, 0, s, dx, dout,
          reinterpret_cast<const TA*>(out_act), p->B, c.hin, c.win, c.cin, c.hout, c.wout, c.cout,
          c.stride)));
    }
    return LSGD_OK;
  }
  dim3 grid((unsigned)((P + 63) / 64), (unsigned)((c.cin + 15) / 16), (unsigned)K);
  const size_t smem = (size_t)c.cout * 9 * 16 * 4;
  RN_LAUNCH((launch_pdl(conv_dgrad_kernel<TA>, grid, 64, smem, s,
      reinterpret_cast<const TA*>(p->dy), reinterpret_cast<const TA*>(Wop) + c.w_off, p->d_pad, dx,
      p->B, c.hin, c.win, c.cin, c.hout, c.wout, c.cout, c.stride, dout,
      reinterpret_cast<const TA*>(out_act))));
  return LSGD_OK;
}

// The weight gradients' deferred partial sums, all in one launch.
lsgd_status flush_sum_jobs(ResNetPlan* p, cudaStream_t s, int64_t* launches) {
  if (p->sum_jobs.empty()) return LSGD_OK;
  SumJobs js{};
  int64_t total = 0;
  for (const SumJob& jb : p->sum_jobs) {
    js.j[js.n] = jb;
    js.j[js.n].begin = total;
    total += (int64_t)jb.G * jb.rows * (jb.cols / 4);
    ++js.n;
  }
  p->sum_jobs.clear();
  RN_LAUNCH((launch_pdl(sum_partials_jobs_v4_kernel, (unsigned)((total + 255) / 256), 256, 0, s, js,
                        total)));
  return LSGD_OK;
}

// Every data gradient's flipped weights for this step, from the bf16 weights, in one launch.
lsgd_status flip_all(ResNetPlan* p, const void* Wop, cudaStream_t s, int64_t* launches) {
  FlipJobs js{};
  int64_t total = 0;
  auto flush = [&]() -> lsgd_status {
    if (total > 0)
      RN_LAUNCH((launch_pdl(flip_jobs_kernel, grid_cap(total, 256), 256, 0, s,
                            reinterpret_cast<const uint16_t*>(Wop), p->d_pad, p->K, js, total)));
    js = FlipJobs{};
    total = 0;
    return LSGD_OK;
  };
  for (size_t i = 0; i < p->wflip.size(); ++i) {
    if (!p->wflip[i]) continue;
    if (js.n == kMaxFlipJobs) {
      const lsgd_status st = flush();  // a deeper network: one launch per table
      if (st != LSGD_OK) return st;
    }
    const ConvL& c = p->convs[i];
    FlipJob& jb = js.j[js.n++];
    jb.w_off = c.w_off;
    jb.dst = p->wflip[i];
    jb.begin = total;
    jb.phases = c.stride == 2 ? 1 : 0;
    jb.n = (jb.phases ? 4 : 1) * (int64_t)p->K * c.cin * 9 * c.cout;
    jb.cin = c.cin;
    jb.cout = c.cout;
    total += jb.n;
  }
  return flush();
}

template <typename TA>
lsgd_status fwd_bwd_impl(ResNetPlan* p, const float* W, const void* Wop, float* Gr,
                         const int32_t* labels, float* loss_mean, cudaStream_t s, int64_t* launches) {
  const int K = p->K, B = p->B;
  p->sum_jobs.clear();
  lsgd_status st = forward_impl<TA>(p, W, Wop, 0, 1, K, s, launches);
  if (st != LSGD_OK) return st;
  RN_CALL(launch_softmax_xent(p->logits, p->C, p->C, labels, K, B, p->dlogits, false, p->C,
                              loss_mean, nullptr, nullptr, s));
  // classifier gradients: G_W = dlogits^T feat, G_b = sum dlogits, dfeat = dlogits W
  {
    GemmArgs g{};
    g.M = p->C;
    g.N = p->F;
    g.Kd = B;
    g.G = K;
    g.A = p->dlogits;
    g.a_rs = 1;
    g.a_cs = p->C;
    g.a_gs = (int64_t)B * p->C;
    g.B = p->feat;
    g.b_rs = p->F;
    g.b_cs = 1;
    g.b_gs = (int64_t)B * p->F;
    g.C = Gr + p->fc_w;
    g.c_rs = p->F;
    g.c_gs = p->d_pad;
    g.epi = EPI_STORE;
    RN_CALL(launch_gemm_simt(g, s));
    RN_CALL(launch_colsum(p->dlogits, false, p->C, K, B, p->C, Gr + p->fc_b, p->d_pad, s));
    GemmArgs h{};
    h.M = B;
    h.N = p->F;
    h.Kd = p->C;
    h.G = K;
    h.A = p->dlogits;
    h.a_rs = p->C;
    h.a_cs = 1;
    h.a_gs = (int64_t)B * p->C;
    h.B = W + p->fc_w;
    h.b_rs = p->F;
    h.b_cs = 1;
    h.b_gs = p->d_pad;
    h.C = p->dfeat;
    h.c_rs = p->F;
    h.c_gs = (int64_t)B * p->F;
    h.epi = EPI_STORE;
    RN_CALL(launch_gemm_simt(h, s));
  }
  const ConvL& last = p->convs.back();
  const int HW = last.hout * last.wout;
  int cur = 0;
  {
    const int64_t n = (int64_t)K * B * HW * p->F;
    RN_LAUNCH((launch_pdl(avgpool_bwd_kernel, grid_cap(n, 256), 256, 0, s, p->dfeat, p->dA[cur], n,
        HW, p->F)));
  }
  const int n_blocks = (int)(p->convs.size() - 1) / 2;
  if (sizeof(TA) == 2) {
    st = flip_all(p, Wop, s, launches);
    if (st != LSGD_OK) return st;
  }
  // partials of the next BatchNorm backward left by the data-gradient epilogue (0: none; the top
  // block's output gradient comes from the pooling's backward)
  int pending = 0;
  for (int j = n_blocks - 1; j >= 0; --j) {
    const int ia = 2 * j + 1, ib = 2 * j + 2;
    const ConvL& ca = p->convs[ia];
    const ConvL& cb = p->convs[ib];
    const void* blk_in = p->act[2 * j];
    // second convolution: BN backward through the block's output ReLU, then its products; its
    // data gradient forms the first convolution's masked gradient and BN sums
    st = bn_backward<TA>(p, cb, ib, p->dA[cur], p->act[ib], W, Gr, s, launches, pending);
    if (st != LSGD_OK) return st;
    st = conv_wgrad<TA>(p, ib, p->act[ia], Gr, s, launches);
    if (st != LSGD_OK) return st;
    int parts_ia = 0;
    st = conv_dgrad<TA>(p, ib, Wop, p->dh, nullptr, nullptr, s, launches, ia, &parts_ia);
    if (st != LSGD_OK) return st;
    // first convolution: BN backward through the inner ReLU, then its products; the data
    // gradient also receives the shortcut's share of the block's output gradient and forms the
    // block input's masked gradient and the BN sums of the convolution that produced it
    st = bn_backward<TA>(p, ca, ia, p->dh, p->act[ia], W, Gr, s, launches, parts_ia);
    if (st != LSGD_OK) return st;
    st = conv_wgrad<TA>(p, ia, blk_in, Gr, s, launches);
    if (st != LSGD_OK) return st;
    st = conv_dgrad<TA>(p, ia, Wop, p->dA[1 - cur], p->dA[cur], p->act[ib], s, launches, 2 * j,
                        &pending);
    if (st != LSGD_OK) return st;
    cur = 1 - cur;
  }
  // stem: BN backward and the weight gradient (no data gradient for the image)
  const ConvL& c0 = p->convs[0];
  st = bn_backward<TA>(p, c0, 0, p->dA[cur], p->act[0], W, Gr, s, launches, pending);
  if (st != LSGD_OK) return st;
  st = conv_wgrad<TA>(p, 0, p->x0, Gr, s, launches);
  if (st != LSGD_OK) return st;
  return flush_sum_jobs(p, s, launches);
}

}  // namespace

size_t batchnorm_stats_scratch_floats(int64_t P, int C, int G) {
  const int64_t nq = (P + kStatChunk - 1) / kStatChunk;
  return (size_t)G * nq * C * 2;
}

size_t conv3x3_scratch_bytes(int mode, int G, int B, int hin, int win, int cin, int cout,
                             int stride) {
  if (mode == 0)
    return cin < 16 ? (conv_x16_elems(G, B, hin, win) + conv_wstem_elems(G, cout)) * 2 : 0;
  return conv_wt_elems(G, cin, cout, stride) * 2;
}

bool conv3x3_tc_route(int mode, int B, int hin, int win, int cin, int cout, int stride) {
  return mode == 0 ? conv_fwd_tc_route(B, hin, win, cin, cout, stride)
                   : conv_dgrad_tc_route(B, hin, win, cin, cout, stride);
}

lsgd_status conv3x3_bf16(int mode, const uint16_t* in, const uint16_t* w, float* out, int G, int B,
                         int hin, int win, int cin, int cout, int stride, void* scratch,
                         cudaStream_t s, std::string* err) {
  std::string e;
  const int64_t w_gs = (int64_t)cout * 9 * cin;
  uint16_t* sc = static_cast<uint16_t*>(scratch);
  lsgd_status st;
  if (mode == 0)
    st = conv_fwd_tc(in, w, w_gs, out, G, B, hin, win, cin, cout, stride, sc,
                     sc ? sc + conv_x16_elems(G, B, hin, win) : nullptr, s, e, nullptr);
  else
    st = conv_dgrad_tc(in, w, w_gs, out, G, B, hin, win, cin, cout, stride, sc, s, e, nullptr);
  if (st != LSGD_OK && err) *err = e;
  return st;
}

size_t conv3x3_bn_scratch_bytes(int G, int B, int hin, int win, int cin, int cout, int stride) {
  int dev = 0, sms = kNumSMs;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
    cudaGetLastError();
    sms = kNumSMs;
  }
  const size_t conv = (conv3x3_scratch_bytes(0, G, B, hin, win, cin, cout, stride) + 15) / 16 * 16;
  return conv + (size_t)4 * (G + 2 * sms) * cout * sizeof(float4);
}

lsgd_status conv3x3_bn_bf16(const uint16_t* in, const uint16_t* w, float* y, float* mean,
                            float* rstd, int G, int B, int hin, int win, int cin, int cout,
                            int stride, void* scratch, cudaStream_t s, std::string* err) {
  std::string e;
  if (cout > 64 || !vec4_ok(cout)) {
    if (err) *err = "the fused statistics take at most 64 output channels";
    return LSGD_EUNSUPPORTED;
  }
  const int64_t w_gs = (int64_t)cout * 9 * cin;
  uint8_t* sc = static_cast<uint8_t*>(scratch);
  const size_t conv = (conv3x3_scratch_bytes(0, G, B, hin, win, cin, cout, stride) + 15) / 16 * 16;
  uint16_t* x16 = conv ? reinterpret_cast<uint16_t*>(sc) : nullptr;
  float4* stats = reinterpret_cast<float4*>(sc + conv);
  int nparts = 0;
  int64_t launches = 0;
  lsgd_status st = conv_fwd_tc(in, w, w_gs, y, G, B, hin, win, cin, cout, stride, x16,
                               x16 ? x16 + conv_x16_elems(G, B, hin, win) : nullptr, s, e,
                               &launches, stats, &nparts);
  if (st == LSGD_OK) {
    launch_pdl(bn_merge_partials_kernel, (G * cout * 32 + 127) / 128, 128, 0, s, stats, nparts, G,
               cout, mean, rstd);
    const cudaError_t ce = cudaGetLastError();
    if (ce != cudaSuccess) {
      e = std::string("statistics merge: ") + cudaGetErrorString(ce);
      st = LSGD_ECUDA;
    }
  }
  if (st != LSGD_OK && err) *err = e;
  return st;
}

size_t conv_wgrad_scratch_floats(int G, int B, int hout, int wout, int cin, int cout, int stride) {
  const int64_t P = (int64_t)B * hout * wout;
  return (size_t)G * conv_wgrad_ctas(cin, stride, wout, G, P) * cout * 9 * cin;
}

cudaError_t launch_conv_wgrad_bf16(const uint16_t* x, const uint16_t* dy, float* dW, int64_t dW_gs,
                                   int G, int B, int hout, int wout, int cin, int cout, int stride,
                                   float* part, cudaStream_t s, int cin_out) {
  return launch_conv_wgrad_impl(x, dy, dW, dW_gs, G, B, hout, wout, cin, cout, stride, part, s,
                                cin_out, nullptr, nullptr);
}

cudaError_t launch_batchnorm_stats(const float* y, int64_t P, int C, int G, float* mean,
                                   float* rstd, float* part, cudaStream_t s) {
  if (P < 1 || C < 1 || C > 256 || G < 1 || G > 65535) return cudaErrorInvalidValue;
  const int64_t nq = (P + kStatChunk - 1) / kStatChunk;
  if (nq > 65535) return cudaErrorInvalidValue;
  const int lanes = std::max(1, 256 / C);
  if (vec4_ok(C))
    launch_pdl(bn_stats_partial_v4_kernel, dim3((unsigned)nq, (unsigned)G), 256, 0, s, y, P, C,
        (int)nq, kStatChunk, part);
  else
    launch_pdl(bn_stats_partial_kernel, dim3((unsigned)nq, (unsigned)G), lanes * C, 0, s, y, P, C,
        (int)nq, kStatChunk, part);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  launch_pdl(bn_stats_finalize_kernel, (G * C * 32 + 127) / 128, 128, 0, s, part, P, C, (int)nq,
      kStatChunk, G, mean, rstd);
  return cudaGetLastError();
}

bool resnet_supported(const lsgd_config& cfg, std::string* why) {
  const lsgd_model& m = cfg.model;
  if (m.in_h < 1 || m.in_w < 1 || m.in_c < 1 || m.n_classes < 1 || m.base_ch < 1 || m.res_blocks < 1) {
    if (why) *why = "ResNet geometry must be positive";
    return false;
  }
  if (m.base_ch * 4 > 64 || m.in_c > 64) {
    if (why) *why = "ResNet channels above 64 are not supported";
    return false;
  }
  if (m.base_ch % 4) {
    if (why) *why = "ResNet base channels must be a multiple of 4";
    return false;
  }
  if ((int64_t)cfg.K * cfg.B_loc * m.in_h * m.in_w * m.base_ch >= (1LL << 31)) {
    if (why) *why = "ResNet activations too large for 32-bit element indexing";
    return false;
  }
  if (cfg.B_loc > 8192 || (int64_t)cfg.B_loc * m.in_h * m.in_w > (1LL << 30)) {
    if (why) *why = "ResNet batch too large";
    return false;
  }
  return true;
}

ResNetPlan* resnet_plan_create(const lsgd_config& cfg) {
  ResNetPlan* p = new ResNetPlan();
  p->cfg = cfg;
  p->K = cfg.K;
  p->B = cfg.B_loc;
  const lsgd_model& m = cfg.model;
  p->H0 = m.in_h;
  p->W0 = m.in_w;
  p->C0 = m.in_c;
  p->C = m.n_classes;
  p->base = m.base_ch;
  p->blocks = m.res_blocks;
  p->bf16 = cfg.precision == LSGD_BF16;
  {
    const char* e = std::getenv("LSGD_FORCE_SIMT");
    p->tc = p->bf16 && tc_available() && !(e && e[0] == '1');
  }
  // layout: canonical order (stem, block convs, fc W, fc b; each conv followed by its BN gamma,
  // beta); padded order puts every BatchNorm parameter after the decayed ones.
  int64_t canon = 0, off = 0;
  int h = p->H0, w = p->W0, ch = p->C0;
  auto add = [&](int cin, int cout, int stride) {
    ConvL c{};
    c.cin = cin;
    c.cout = cout;
    c.stride = stride;
    c.hin = h;
    c.win = w;
    c.hout = (h - 1) / stride + 1;
    c.wout = (w - 1) / stride + 1;
    c.cw = canon;
    canon += (int64_t)cout * 9 * cin;
    c.cg = canon;
    canon += cout;
    c.cb = canon;
    canon += cout;
    c.w_off = off;
    off = rup(off + (int64_t)cout * 9 * cin, 64);
    h = c.hout;
    w = c.wout;
    p->convs.push_back(c);
  };
  add(ch, p->base, 1);
  ch = p->base;
  for (int st = 0; st < 3; ++st) {
    const int cout = p->base << st;
    for (int b = 0; b < p->blocks; ++b) {
      add(ch, cout, (st > 0 && b == 0) ? 2 : 1);
      add(cout, cout, 1);
      ch = cout;
    }
  }
  p->F = ch;
  p->c_fc_w = canon;
  canon += (int64_t)p->C * p->F;
  p->c_fc_b = canon;
  canon += p->C;
  p->fc_w = off;
  off = rup(off + (int64_t)p->C * p->F, 64);
  p->fc_b = off;
  off = rup(off + p->C, 64);
  p->decay_end = off;
  for (ConvL& c : p->convs) {
    c.g_off = off;
    off = rup(off + c.cout, 64);
    c.b_off = off;
    off = rup(off + c.cout, 64);
  }
  p->d = canon;
  p->d_pad = rup(off, 64);
  int64_t mx = (int64_t)p->B * p->H0 * p->W0 * p->C0;
  for (const ConvL& c : p->convs) mx = std::max(mx, (int64_t)p->B * c.hout * c.wout * c.cout);
  p->max_act = mx * p->K;
  return p;
}

void resnet_destroy(ResNetPlan* p) { delete p; }
int64_t resnet_num_params(const ResNetPlan* p) { return p->d; }
int64_t resnet_d_pad(const ResNetPlan* p) { return p->d_pad; }

void resnet_segments(const ResNetPlan* p, const std::function<void(int64_t, int64_t, int64_t)>& f) {
  for (const ConvL& c : p->convs) {
    f(c.cw, c.w_off, (int64_t)c.cout * 9 * c.cin);
    f(c.cg, c.g_off, c.cout);
    f(c.cb, c.b_off, c.cout);
  }
  f(p->c_fc_w, p->fc_w, (int64_t)p->C * p->F);
  f(p->c_fc_b, p->fc_b, p->C);
}

void resnet_decay_region(const ResNetPlan* p, int64_t* period, int64_t* decay_end) {
  *period = p->d_pad;
  *decay_end = p->decay_end;
}

lsgd_status resnet_alloc(ResNetPlan* p, const std::function<void*(size_t)>& alloc) {
  const int K = p->K, B = p->B;
  const size_t e = esz(p);
  p->x0 = alloc((size_t)K * B * p->H0 * p->W0 * p->C0 * e);
  size_t part = 0, colT = 0, wt = 0, wt4 = 0;
  p->stem16 = stem16_ok(p, p->convs[0]);
  if (p->stem16) {
    const ConvL& c0 = p->convs[0];
    p->x16 = (uint16_t*)alloc((size_t)K * B * c0.hin * c0.win * 16 * 2);
    p->wstem = (uint16_t*)alloc((size_t)K * c0.cout * 9 * 16 * 2);
    if (!p->x16 || !p->wstem) return LSGD_ENOMEM;
    const int64_t P0 = (int64_t)B * c0.hout * c0.wout;
    part = std::max(part, (size_t)K * conv_wgrad_ctas(16, 1, c0.wout, K, P0) * c0.cout * 9 * 16);
  }
  for (const ConvL& c : p->convs) {
    const int64_t n = (int64_t)K * B * c.hout * c.wout * c.cout;
    p->y.push_back((float*)alloc((size_t)n * 4));
    p->act.push_back(alloc((size_t)n * e));
    p->mean.push_back((float*)alloc((size_t)K * c.cout * 4));
    p->rstd.push_back((float*)alloc((size_t)K * c.cout * 4));
    const int64_t P = (int64_t)B * c.hout * c.wout;
    const int64_t nq_s = (P + kRnChunk - 1) / kRnChunk;
    const int64_t nq_w = (P + kWgradChunk - 1) / kWgradChunk;
    part = std::max(part, (size_t)(K * nq_s * c.cout * 2));
    part = std::max(part, (size_t)(K * nq_w * c.cout * 9 * c.cin));
    float* wp = nullptr;
    if (conv_on_tc(p, c)) {
      const int Kc = col_ld(c);
      if (wgrad_tc(p, c)) {
        const int cpr = conv_wgrad_ctas(c.cin, c.stride, c.wout, K, P);
        part = std::max(part, (size_t)K * cpr * c.cout * 9 * c.cin);
        if (!(&c == &p->convs[0] && p->stem16)) {
          wp = (float*)alloc((size_t)K * cpr * c.cout * 9 * c.cin * 4);
          if (!wp) return LSGD_ENOMEM;
        }
      } else {
        const int tiles = ((Kc + 63) / 64) * K;
        const int splits = tc_valid_splits((int)P, std::max(1, (4 * kNumSMs + tiles - 1) / tiles));
        part = std::max(part, (size_t)K * splits * c.cout * Kc);
      }
      if (needs_col(p, c) && !(&c == &p->convs[0] && p->stem16)) {
        p->col.push_back((uint16_t*)alloc((size_t)K * P * Kc * 2));
        if (!p->col.back()) return LSGD_ENOMEM;
      } else {
        p->col.push_back(nullptr);
      }
      if (c.cin % 8 == 0) {
        if (phase_dgrad_ok(p, c))
          wt4 = std::max(wt4, (size_t)4 * K * c.cin * 9 * c.cout);
        else if (!(c.stride == 1 && implicit_conv_ok(c.cout, 1, c.hin, c.win)))
          colT = std::max(colT, (size_t)K * B * c.hin * c.win * 9 * c.cout);
        wt = std::max(wt, (size_t)K * c.cin * 9 * c.cout);
      } else {
        wt = std::max(wt, (size_t)K * c.cout * Kc);
      }
    } else {
      p->col.push_back(nullptr);
    }
    p->wpart.push_back(wp);
    // this convolution's data gradient on the persistent implicit kernel: its own flipped weights
    uint16_t* wf = nullptr;
    if (&c != &p->convs[0] && conv_on_tc(p, c)) {
      const int64_t Pd = (int64_t)B * c.hin * c.win;
      const size_t per = (size_t)K * c.cin * 9 * c.cout;
      const bool plain = c.stride == 1 && implicit_conv_ok(c.cout, 1, c.hin, c.win) &&
                         persistent_conv_ok(c.cin, Pd);
      const bool phases = !plain && phase_dgrad_ok(p, c);
      if (plain || phases) {
        wf = (uint16_t*)alloc((phases ? 4 : 1) * per * 2);
        if (!wf) return LSGD_ENOMEM;
      }
    }
    p->wflip.push_back(wf);
  }
  if (colT) {
    p->colT = (uint16_t*)alloc(colT * 2);
    if (!p->colT) return LSGD_ENOMEM;
  }
  if (wt) {
    p->wt = (uint16_t*)alloc(wt * 2);
    if (!p->wt) return LSGD_ENOMEM;
  }
  if (wt4) {
    p->wt4 = (uint16_t*)alloc(wt4 * 2);
    if (!p->wt4) return LSGD_ENOMEM;
  }
  p->part_floats = part;
  p->part = (float*)alloc(part * 4);
  p->feat = (float*)alloc((size_t)K * B * p->F * 4);
  p->dfeat = (float*)alloc((size_t)K * B * p->F * 4);
  p->logits = (float*)alloc((size_t)K * B * p->C * 4);
  p->dlogits = (float*)alloc((size_t)K * B * p->C * 4);
  p->dA[0] = (float*)alloc((size_t)p->max_act * 4);
  p->dA[1] = (float*)alloc((size_t)p->max_act * 4);
  p->dh = (float*)alloc((size_t)p->max_act * 4);
  p->dy = alloc((size_t)p->max_act * e);
  p->s12 = (float*)alloc((size_t)K * 2 * 64 * 4);
  if (p->tc) {
    // at most max(K, 2 SMs) CTAs over all replicas (launch_conv_tc), four partials of 64
    // channels each
    int dev = 0, sms = kNumSMs;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return LSGD_ECUDA;
    p->cstats = (float4*)alloc((size_t)4 * (K + 2 * sms) * 64 * sizeof(float4));
    // four phases x four warps x (CTAs over all replicas <= max(K, 2 SMs)) partials of 64 channels
    p->bpart = (float2*)alloc((size_t)16 * (K + 2 * sms) * 64 * sizeof(float2));
    if (!p->cstats || !p->bpart) return LSGD_ENOMEM;
  }
  if (!p->x0 || !p->part || !p->feat || !p->dfeat || !p->logits || !p->dlogits || !p->dA[0] ||
      !p->dA[1] || !p->dh || !p->dy || !p->s12)
    return LSGD_ENOMEM;
  for (size_t i = 0; i < p->convs.size(); ++i)
    if (!p->y[i] || !p->act[i] || !p->mean[i] || !p->rstd[i]) return LSGD_ENOMEM;
  return LSGD_OK;
}

// He initialisation of the convolutions (fan-in 9 Cin), N(0, 0.01^2) for the classifier, zero
// biases, BN gamma = 1 and beta = 0 (Sec. A.2); replica 0, broadcast by the caller.
lsgd_status resnet_init_params(ResNetPlan* p, float* W, uint64_t seed, cudaStream_t s,
                               int64_t* launches) {
  if (p->cfg.model.init != LSGD_INIT_HE) return LSGD_OK;  // all zeros
  uint32_t tensor = 0;
  for (const ConvL& c : p->convs) {
    RN_CALL(launch_init_normal(W + c.w_off, (int64_t)c.cout * 9 * c.cin, std::sqrt(2.0 / (9.0 * c.cin)),
                               seed, tensor, s));
    ++tensor;
    RN_CALL(launch_fill(W + c.g_off, c.cout, 1.0f, s));
  }
  RN_CALL(launch_init_normal(W + p->fc_w, (int64_t)p->C * p->F, 0.01, seed, tensor, s));
  return LSGD_OK;
}

lsgd_status resnet_forward_backward(ResNetPlan* p, const float* W, const uint16_t* Wb, float* G,
                                    int64_t d_pad, const int32_t* labels, float* loss_mean,
                                    cudaStream_t s, int64_t* launches) {
  (void)d_pad;
  if (p->bf16) return fwd_bwd_impl<uint16_t>(p, W, Wb, G, labels, loss_mean, s, launches);
  return fwd_bwd_impl<float>(p, W, W, G, labels, loss_mean, s, launches);
}

lsgd_status resnet_eval(ResNetPlan* p, const float* W, const uint16_t* Wb, int64_t d_pad, int k,
                        int groups, const int32_t* labels, float* row_loss, cudaStream_t s,
                        int64_t* launches) {
  (void)d_pad;
  lsgd_status st = p->bf16 ? forward_impl<uint16_t>(p, W, Wb, k, 0, groups, s, launches)
                           : forward_impl<float>(p, W, W, k, 0, groups, s, launches);
  if (st != LSGD_OK) return st;
  RN_CALL(launch_softmax_xent(p->logits, p->C, p->C, labels, groups, p->B, nullptr, false, p->C,
                              nullptr, nullptr, row_loss, s));
  return LSGD_OK;
}

void* resnet_input(ResNetPlan* p) { return p->x0; }
const char* resnet_last_error(const ResNetPlan* p) { return p ? p->err.c_str() : ""; }

}  // namespace lsgd
