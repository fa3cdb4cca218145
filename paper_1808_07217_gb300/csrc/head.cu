// Classifier head of a dense network in bf16 mode: the last layer (C <= 16 classes) and its loss in
// two kernels instead of five (forward product, softmax cross-entropy, data gradient, weight
// gradient + update, bias gradient + update).  Its products are tiny (C outputs per row), so they
// run on the SIMT cores straight from the bf16 operands the tensor-core path would use: the stored
// activation a, the bf16 shadow of W, and the bf16-rounded logits gradient dZ (Eq. 2's local
// gradient of the softmax cross-entropy loss), with fp32 accumulation.
//
//   head_forward_kernel   z = a W^T + b, l = logsumexp(z) - z_y, dZ = (softmax(z) - onehot(y)) / B,
//                         and dA = (dZ W) * (a > 0) for the layer below, row by row
//   head_backward_kernel  per 64-column block of W: gW = dZ^T a, the bias gradient of the layer
//                         below for those 64 columns (sum over rows of dA), and for block 0
//                         gb = sum_j dZ_j and the mean loss; then the local update of those
//                         parameters (fused mode) or the gradients (else)
#include "../../include/lsgd.h"
#include "common.cuh"
#include "lsgd_internal.h"

namespace lsgd {
namespace {

constexpr int kHeadRowsPerWarp = 1;
constexpr int kHeadRowsPerCta = 8 * kHeadRowsPerWarp;
constexpr int kHeadCols = 64;   // W columns per backward CTA (eight chunks of eight)

__device__ __forceinline__ void bf16x8_to_f32(const uint4 v, float (&f)[8]) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    f[2 * i] = bf2f((uint16_t)(w[i] & 0xffffu));
    f[2 * i + 1] = bf2f((uint16_t)(w[i] >> 16));
  }
}

// A CTA takes 8 rows of one replica (one per warp) with the replica's weights staged in shared
// memory: the forward product (lanes split the reduction, a butterfly closes it), the loss and the
// bf16 logits gradient, then the data gradient of the same rows for the layer below, read from the
// rounded dZ and the still un-updated weights.
template <int CMAX>
__global__ void __launch_bounds__(256) head_forward_kernel(HeadArgs h) {
  pdl_begin();
  extern __shared__ uint4 wsm[];  // [C][in / 8] this replica's bf16 weights
  const int g = blockIdx.y, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int C = h.C, chunks = h.in / 8;
  {
    const uint4* Wg = reinterpret_cast<const uint4*>(h.Wb + (int64_t)g * h.rep_stride + h.w_off);
#pragma unroll 4
    for (int i = threadIdx.x; i < C * chunks; i += blockDim.x) wsm[i] = __ldg(Wg + i);
  }
  __syncthreads();
  const int jw = blockIdx.x * kHeadRowsPerCta + warp * kHeadRowsPerWarp;
  if (jw >= h.B) return;
  const int nr = min(kHeadRowsPerWarp, h.B - jw);
  const uint16_t* arow[kHeadRowsPerWarp];
#pragma unroll
  for (int r = 0; r < kHeadRowsPerWarp; ++r)
    arow[r] = h.act + ((int64_t)g * h.B + jw + min(r, nr - 1)) * h.ld_in;
  float acc[kHeadRowsPerWarp][CMAX];
#pragma unroll
  for (int r = 0; r < kHeadRowsPerWarp; ++r)
#pragma unroll
    for (int c = 0; c < CMAX; ++c) acc[r][c] = 0.f;
#pragma unroll 2
  for (int ch = lane; ch < chunks; ch += 32) {
    uint4 araw[kHeadRowsPerWarp];
#pragma unroll
    for (int r = 0; r < kHeadRowsPerWarp; ++r) araw[r] = *reinterpret_cast<const uint4*>(arow[r] + ch * 8);
    float x[kHeadRowsPerWarp][8];
#pragma unroll
    for (int r = 0; r < kHeadRowsPerWarp; ++r) bf16x8_to_f32(araw[r], x[r]);
#pragma unroll
    for (int c = 0; c < CMAX; ++c) {
      if (c < C) {
        float wv[8];
        bf16x8_to_f32(wsm[c * chunks + ch], wv);
#pragma unroll
        for (int r = 0; r < kHeadRowsPerWarp; ++r)
#pragma unroll
          for (int i = 0; i < 8; ++i) acc[r][c] = fmaf(x[r][i], wv[i], acc[r][c]);
      }
    }
  }
#pragma unroll
  for (int r = 0; r < kHeadRowsPerWarp; ++r)
#pragma unroll
    for (int c = 0; c < CMAX; ++c)
      if (c < C) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) acc[r][c] += __shfl_xor_sync(0xffffffffu, acc[r][c], o);
      }
  const float* bias = h.W + (int64_t)g * h.rep_stride + h.b_off;
  const float inv_b = 1.0f / (float)h.B;
  // softmax cross-entropy per row; every lane keeps the row's rounded dZ for the data gradient
#pragma unroll
  for (int r = 0; r < kHeadRowsPerWarp; ++r) {
    float mx = -INFINITY;
#pragma unroll
    for (int c = 0; c < CMAX; ++c) {
      acc[r][c] = c < C ? acc[r][c] + bias[c] : -INFINITY;
      mx = fmaxf(mx, acc[r][c]);
    }
    float se = 0.f;
#pragma unroll
    for (int c = 0; c < CMAX; ++c)
      if (c < C) se += expf(acc[r][c] - mx);
    const float lse = mx + logf(se);
    const int64_t row = (int64_t)g * h.B + jw + r;
    const int y = r < nr ? h.labels[row] : -1;
    float zy = 0.f;
#pragma unroll
    for (int c = 0; c < CMAX; ++c) {
      if (c == y) zy = acc[r][c];
      const float p = c < C ? expf(acc[r][c] - lse) : 0.f;
      const uint16_t q = f2bf((p - (c == y ? 1.f : 0.f)) * inv_b);
      if (r < nr && c < C && c == lane) h.dz[row * h.ld_dz + c] = q;
      acc[r][c] = c < C ? bf2f(q) : 0.f;  // acc now holds the row's rounded dZ
    }
    if (r < nr && lane == 0) h.row_loss[row] = lse - zy;
  }
  if (!h.dz_prev) return;
  for (int ch = lane; ch < chunks; ch += 32) {
#pragma unroll
    for (int r = 0; r < kHeadRowsPerWarp; ++r) {
      if (r >= nr) break;
      float a[8], dA[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
      bf16x8_to_f32(*reinterpret_cast<const uint4*>(arow[r] + ch * 8), a);
#pragma unroll
      for (int c = 0; c < CMAX; ++c) {
        if (c < C) {
          float wv[8];
          bf16x8_to_f32(wsm[c * chunks + ch], wv);
#pragma unroll
          for (int i = 0; i < 8; ++i) dA[i] = fmaf(acc[r][c], wv[i], dA[i]);
        }
      }
      uint32_t o[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float v0 = a[2 * i] > 0.f ? dA[2 * i] : 0.f;
        const float v1 = a[2 * i + 1] > 0.f ? dA[2 * i + 1] : 0.f;
        o[i] = (uint32_t)f2bf(v0) | ((uint32_t)f2bf(v1) << 16);
      }
      const int64_t row = (int64_t)g * h.B + jw + r;
      *reinterpret_cast<uint4*>(h.dz_prev + row * h.ld_dz_prev + ch * 8) =
          make_uint4(o[0], o[1], o[2], o[3]);
    }
  }
}

// Weight and bias gradients of the head for one replica and a block of 64 columns.  Warp w sums
// rows w, w + 8, ...; lane = (chunk of eight columns, class group of CMAX / 4 classes), so a lane
// holds 8 x CMAX / 4 partial sums, which the eight warps then add in warp order through shared
// memory.  Then the local update of those parameters (fused mode) or the gradient (else).
template <int CMAX>
__global__ void __launch_bounds__(256) head_backward_kernel(HeadArgs h) {
  pdl_begin();
  constexpr int CG = CMAX / 4;              // classes per lane
  extern __shared__ float hsm[];
  float* dzs = hsm;                         // [B][CMAX] the bf16 logits gradient as fp32
  float* part = hsm + (size_t)h.B * CMAX;   // [8 warps][CMAX][64] partial sums
  const int g = blockIdx.y, n0 = blockIdx.x * kHeadCols;
  const int C = h.C, t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const int ch = lane & 7, cg = lane >> 3;  // chunk, class group
  const int64_t rep = (int64_t)g * h.rep_stride;
  for (int j = t; j < h.B; j += blockDim.x) {
    const uint16_t* src = h.dz + ((int64_t)g * h.B + j) * h.ld_dz;
    uint16_t v[CMAX];
#pragma unroll
    for (int c = 0; c < CMAX; ++c) v[c] = c < C ? src[c] : (uint16_t)0;
#pragma unroll
    for (int c = 0; c < CMAX; ++c) dzs[j * CMAX + c] = c < C ? bf2f(v[c]) : 0.f;
  }
  __syncthreads();
  const int nb = n0 + ch * 8;
  const bool col_ok = nb < h.in;
  float acc[CG][8];
#pragma unroll
  for (int q = 0; q < CG; ++q)
#pragma unroll
    for (int i = 0; i < 8; ++i) acc[q][i] = 0.f;
  if (col_ok) {
#pragma unroll 4
    for (int j = warp; j < h.B; j += 8) {
      float a[8];
      bf16x8_to_f32(*reinterpret_cast<const uint4*>(h.act + ((int64_t)g * h.B + j) * h.ld_in + nb), a);
#pragma unroll
      for (int q = 0; q < CG; ++q) {
        const float d = dzs[j * CMAX + cg * CG + q];
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[q][i] = fmaf(d, a[i], acc[q][i]);
      }
    }
  }
#pragma unroll
  for (int q = 0; q < CG; ++q)
#pragma unroll
    for (int i = 0; i < 8; ++i) part[(warp * CMAX + cg * CG + q) * kHeadCols + ch * 8 + i] = acc[q][i];
  __syncthreads();
  const SgdParams& sp = h.sgd;
  const bool sg = sp.sign != 0;
  // output o = (class c, column n): consecutive threads take consecutive columns of a class row
  for (int o = t; o < C * kHeadCols; o += blockDim.x) {
    const int c = o / kHeadCols, n = o % kHeadCols;
    if (n0 + n >= h.in) continue;
    float s = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) s += part[(w * CMAX + c) * kHeadCols + n];
    const int64_t k = rep + h.w_off + (int64_t)c * h.in + n0 + n;
    if (!h.fused) {
      h.grad[k] = s;
      continue;
    }
    float w = sp.w[k], u = sp.u ? sp.u[k] : 0.f;
    if (sp.mom == 0.f)
      sgd_elem<false, false>(w, u, s, sp.lr, 0.f, sp.wd, sg);
    else if (sp.nesterov)
      sgd_elem<true, true>(w, u, s, sp.lr, sp.mom, sp.wd, sg);
    else
      sgd_elem<true, false>(w, u, s, sp.lr, sp.mom, sp.wd, sg);
    sp.w[k] = w;
    if (sp.u) sp.u[k] = u;
    if (sp.wb) sp.wb[k] = f2bf(w);
  }
  // the layer below: its bias gradient for this block's 64 columns = sum over rows of the bf16
  // data gradient the forward kernel stored (four row quarters, then added in quarter order)
  if (h.b_prev_off >= 0 && h.dz_prev) {
    __syncthreads();  // part[] is free again
    const int n = t & (kHeadCols - 1), qtr = t / kHeadCols;  // 4 quarters of the rows
    float s = 0.f;
    if (n0 + n < h.in) {
      const int rows = (h.B + 3) / 4, j0 = qtr * rows, j1 = min(h.B, j0 + rows);
      const uint16_t* col = h.dz_prev + ((int64_t)g * h.B) * h.ld_dz_prev + n0 + n;
      int j = j0;
      // eight rows' loads in flight, then added in row order (the same sum as one at a time)
      for (; j + 8 <= j1; j += 8) {
        float v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) v[u] = bf2f(col[(int64_t)(j + u) * h.ld_dz_prev]);
#pragma unroll
        for (int u = 0; u < 8; ++u) s += v[u];
      }
      for (; j < j1; ++j) s += bf2f(col[(int64_t)j * h.ld_dz_prev]);
    }
    part[qtr * kHeadCols + n] = s;
    __syncthreads();
    if (t < kHeadCols && n0 + t < h.in) {
      const float gb = ((part[t] + part[kHeadCols + t]) + part[2 * kHeadCols + t]) +
                       part[3 * kHeadCols + t];
      const int64_t k = rep + h.b_prev_off + n0 + t;
      if (!h.fused) {
        h.grad[k] = gb;
      } else {
        float w = sp.w[k], u = sp.u ? sp.u[k] : 0.f;
        if (sp.mom == 0.f)
          sgd_elem<false, false>(w, u, gb, sp.lr, 0.f, sp.wd, sg);
        else if (sp.nesterov)
          sgd_elem<true, true>(w, u, gb, sp.lr, sp.mom, sp.wd, sg);
        else
          sgd_elem<true, false>(w, u, gb, sp.lr, sp.mom, sp.wd, sg);
        sp.w[k] = w;
        if (sp.u) sp.u[k] = u;
        if (sp.wb) sp.wb[k] = f2bf(w);
      }
    }
  }
  // bias gradient (one warp per class, a fixed butterfly over rows) and the mean loss (warp 7):
  // the first column block of each replica
  if (blockIdx.x == 0) {
    for (int c = warp; c < C; c += 7) {
      if (warp == 7) break;
      float s = 0.f;
      for (int j = lane; j < h.B; j += 32) s += dzs[j * CMAX + c];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
      if (lane == 0) {
        const int64_t k = rep + h.b_off + c;
        if (!h.fused) {
          h.grad[k] = s;
        } else {
          float w = sp.w[k], u = sp.u ? sp.u[k] : 0.f;
          if (sp.mom == 0.f)
            sgd_elem<false, false>(w, u, s, sp.lr, 0.f, sp.wd, sg);
          else if (sp.nesterov)
            sgd_elem<true, true>(w, u, s, sp.lr, sp.mom, sp.wd, sg);
          else
            sgd_elem<true, false>(w, u, s, sp.lr, sp.mom, sp.wd, sg);
          sp.w[k] = w;
          if (sp.u) sp.u[k] = u;
          if (sp.wb) sp.wb[k] = f2bf(w);
        }
      }
    }
    if (warp == 7 && h.loss_mean) {
      float s = 0.f;
      for (int j = lane; j < h.B; j += 32) s += h.row_loss[(int64_t)g * h.B + j];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
      if (lane == 0) h.loss_mean[g] = s / (float)h.B;
    }
  }
}

}  // namespace

bool head_supported(int C, int B, int in) {
  return C >= 1 && C <= kHeadMaxClasses && B >= 1 && B <= 1024 && in % 8 == 0 &&
         (size_t)C * in * 2 <= 48 * 1024 &&                             // forward: the weights
         (size_t)(B + 8 * kHeadCols) * kHeadMaxClasses * 4 <= 96 * 1024;  // backward: dZ + partials
}

namespace {
template <int CMAX>
cudaError_t head_launch(const HeadArgs& h, bool backward, cudaStream_t stream) {
  if (!backward) {
    const dim3 grid((h.B + kHeadRowsPerCta - 1) / kHeadRowsPerCta, h.reps);
    return launch_pdl(head_forward_kernel<CMAX>, grid, dim3(256), (size_t)h.C * h.in * 2, stream, h);
  }
  const size_t smem = (size_t)(h.B + 8 * kHeadCols) * CMAX * sizeof(float);
  static int attr_dev = -1;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (attr_dev != dev) {
    e = cudaFuncSetAttribute(head_backward_kernel<CMAX>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             96 * 1024);
    if (e != cudaSuccess) return e;
    attr_dev = dev;
  }
  const dim3 grid((h.in + kHeadCols - 1) / kHeadCols, h.reps);
  return launch_pdl(head_backward_kernel<CMAX>, grid, dim3(256), smem, stream, h);
}
}  // namespace

cudaError_t launch_head_forward(const HeadArgs& h, cudaStream_t stream) {
  if (!head_supported(h.C, h.B, h.in) || h.reps < 1 || h.reps > 65535) return cudaErrorInvalidValue;
  if (h.C <= 8) return head_launch<8>(h, false, stream);
  if (h.C <= 12) return head_launch<12>(h, false, stream);
  return head_launch<16>(h, false, stream);
}

cudaError_t launch_head_backward(const HeadArgs& h, cudaStream_t stream) {
  if (!head_supported(h.C, h.B, h.in) || h.reps < 1 || h.reps > 65535) return cudaErrorInvalidValue;
  if (h.fused ? !h.sgd.w || (h.sgd.mom != 0.f && !h.sgd.u) : !h.grad) return cudaErrorInvalidValue;
  if (h.C <= 8) return head_launch<8>(h, true, stream);
  if (h.C <= 12) return head_launch<12>(h, true, stream);
  return head_launch<16>(h, true, stream);
}

}  // namespace lsgd
