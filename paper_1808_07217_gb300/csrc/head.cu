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

constexpr int kHeadThreads = 256;
constexpr int kHeadRowsPerCta = kHeadThreads / 32;  // one row per warp in the forward kernel
constexpr int kHeadCols = 64;        // W columns per backward CTA (eight chunks of eight)
constexpr int kHeadChunksPerLane = 4;  // forward: 8-column chunks of the row a lane holds in registers

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
// rounded dZ and the still un-updated weights.  The work per row is tiny, so the kernel's time is
// its chain of memory round trips: the row (up to 32 x kHeadChunksPerLane chunks, kept in
// registers for both products), the label and the bias are all requested before the weights are
// staged, and one round trip serves them all.
template <int CMAX>
__global__ void __launch_bounds__(kHeadThreads) head_forward_kernel(HeadArgs h) {
  pdl_begin();
  extern __shared__ uint4 wsm[];  // [C][in / 8] this replica's bf16 weights
  const int g = blockIdx.y, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int C = h.C, chunks = h.in / 8;
  const int j = blockIdx.x * kHeadRowsPerCta + warp;  // this warp's row
  const bool row_ok = j < h.B;
  const int64_t row = (int64_t)g * h.B + (row_ok ? j : 0);
  const uint16_t* arow = h.act + row * h.ld_in;
  uint4 araw[kHeadChunksPerLane];
#pragma unroll
  for (int q = 0; q < kHeadChunksPerLane; ++q) {
    const int ch = lane + 32 * q;
    araw[q] = (row_ok && ch < chunks) ? *reinterpret_cast<const uint4*>(arow + ch * 8)
                                      : make_uint4(0u, 0u, 0u, 0u);
  }
  const float* bias = h.W + (int64_t)g * h.rep_stride + h.b_off;
  float bv[CMAX];
#pragma unroll
  for (int c = 0; c < CMAX; ++c) bv[c] = c < C ? bias[c] : 0.f;
  const int y = row_ok ? h.labels[row] : -1;
  {
    const uint4* Wg = reinterpret_cast<const uint4*>(h.Wb + (int64_t)g * h.rep_stride + h.w_off);
#pragma unroll 8
    for (int i = threadIdx.x; i < C * chunks; i += kHeadThreads) wsm[i] = __ldg(Wg + i);
  }
  __syncthreads();
  if (!row_ok) return;
  // z = a W^T: lane-partial sums over chunks lane, lane + 32, ... in that order
  float acc[CMAX];
#pragma unroll
  for (int c = 0; c < CMAX; ++c) acc[c] = 0.f;
  auto dot = [&](const uint4 raw, int ch) {
    float x[8];
    bf16x8_to_f32(raw, x);
#pragma unroll
    for (int c = 0; c < CMAX; ++c) {
      if (c < C) {
        float wv[8];
        bf16x8_to_f32(wsm[c * chunks + ch], wv);
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[c] = fmaf(x[i], wv[i], acc[c]);
      }
    }
  };
#pragma unroll
  for (int q = 0; q < kHeadChunksPerLane; ++q)
    if (lane + 32 * q < chunks) dot(araw[q], lane + 32 * q);
  for (int ch = lane + 32 * kHeadChunksPerLane; ch < chunks; ch += 32)
    dot(*reinterpret_cast<const uint4*>(arow + ch * 8), ch);
#pragma unroll
  for (int c = 0; c < CMAX; ++c)
    if (c < C) {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) acc[c] += __shfl_xor_sync(0xffffffffu, acc[c], o);
    }
  const float inv_b = 1.0f / (float)h.B;
  // softmax cross-entropy of the row; every lane keeps the row's rounded dZ for the data gradient
  float mx = -INFINITY;
#pragma unroll
  for (int c = 0; c < CMAX; ++c) {
    acc[c] = c < C ? acc[c] + bv[c] : -INFINITY;
    mx = fmaxf(mx, acc[c]);
  }
  float se = 0.f;
#pragma unroll
  for (int c = 0; c < CMAX; ++c)
    if (c < C) se += expf(acc[c] - mx);
  const float lse = mx + logf(se);
  float zy = 0.f;
#pragma unroll
  for (int c = 0; c < CMAX; ++c) {
    if (c == y) zy = acc[c];
    const float p = c < C ? expf(acc[c] - lse) : 0.f;
    const uint16_t q = f2bf((p - (c == y ? 1.f : 0.f)) * inv_b);
    if (c < C && c == lane) h.dz[row * h.ld_dz + c] = q;
    acc[c] = c < C ? bf2f(q) : 0.f;  // acc now holds the row's rounded dZ
  }
  if (lane == 0) h.row_loss[row] = lse - zy;
  if (!h.dz_prev) return;
  // dA = (dZ W) * (a > 0), chunk by chunk, stored as bf16
  auto dgrad = [&](const uint4 raw, int ch) {
    float a[8], dA[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    bf16x8_to_f32(raw, a);
#pragma unroll
    for (int c = 0; c < CMAX; ++c) {
      if (c < C) {
        float wv[8];
        bf16x8_to_f32(wsm[c * chunks + ch], wv);
#pragma unroll
        for (int i = 0; i < 8; ++i) dA[i] = fmaf(acc[c], wv[i], dA[i]);
      }
    }
    uint32_t o[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float v0 = a[2 * i] > 0.f ? dA[2 * i] : 0.f;
      const float v1 = a[2 * i + 1] > 0.f ? dA[2 * i + 1] : 0.f;
      o[i] = (uint32_t)f2bf(v0) | ((uint32_t)f2bf(v1) << 16);
    }
    *reinterpret_cast<uint4*>(h.dz_prev + row * h.ld_dz_prev + ch * 8) = make_uint4(o[0], o[1], o[2], o[3]);
  };
#pragma unroll
  for (int q = 0; q < kHeadChunksPerLane; ++q)
    if (lane + 32 * q < chunks) dgrad(araw[q], lane + 32 * q);
  for (int ch = lane + 32 * kHeadChunksPerLane; ch < chunks; ch += 32)
    dgrad(*reinterpret_cast<const uint4*>(arow + ch * 8), ch);
}

// Weight and bias gradients of the head for one replica and a block of 64 columns.  Warp w sums
// rows w, w + 8, ...; lane = (chunk of eight columns, class group of CMAX / 4 classes), so a lane
// holds 8 x CMAX / 4 partial sums, which the eight warps then add in warp order through shared
// memory.  Then the local update of those parameters (fused mode) or the gradient (else).
//
// Like the forward kernel this one is a chain of memory round trips, so each load is issued as
// soon as nothing orders it: the parameters a thread updates in place (no other thread touches
// them), the first rows' activations and the logits gradient in the first wave, the next rows'
// activations while the first are summed, the layer below's data gradient while the partial sums
// are exchanged.
template <int CMAX>
__global__ void __launch_bounds__(kHeadThreads, 2) head_backward_kernel(HeadArgs h) {
  pdl_begin();
  constexpr int CG = CMAX / 4;  // classes per lane; also updated outputs per thread
  constexpr int RB = CMAX > 12 ? 4 : 8;  // rows per warp whose activation loads fly together
  constexpr int PR = 4;         // rows per thread of the layer-below bias sums in flight together
  static_assert(CMAX * kHeadCols == CG * kHeadThreads, "one update output per thread and class group");
  extern __shared__ float hsm[];
  float* dzs = hsm;                        // [B][CMAX] the bf16 logits gradient as fp32
  float* part = hsm + (size_t)h.B * CMAX;  // [8 warps][CMAX][64] partial sums
  const int g = blockIdx.y, n0 = blockIdx.x * kHeadCols;
  const int C = h.C, t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const int ch = lane & 7, cg = lane >> 3;  // chunk, class group
  const int64_t rep = (int64_t)g * h.rep_stride;
  const SgdParams& sp = h.sgd;
  const bool fused = h.fused != 0;
  const bool sg = sp.sign != 0;
  auto update = [&](float& w, float& u, float gr) {
    if (sp.mom == 0.f)
      sgd_elem<false, false>(w, u, gr, sp.lr, 0.f, sp.wd, sg);
    else if (sp.nesterov)
      sgd_elem<true, true>(w, u, gr, sp.lr, sp.mom, sp.wd, sg);
    else
      sgd_elem<true, false>(w, u, gr, sp.lr, sp.mom, sp.wd, sg);
  };
  auto store = [&](int64_t k, float w, float u) {
    sp.w[k] = w;
    if (sp.u) sp.u[k] = u;
    if (sp.wb) sp.wb[k] = f2bf(w);
  };

  // ---- first wave of loads ----
  const int nb = n0 + ch * 8;
  const bool col_ok = nb < h.in;
  const uint16_t* abase = h.act + (int64_t)g * h.B * h.ld_in + nb;
  auto load_rows = [&](uint4 (&dst)[RB], int j0) {
#pragma unroll
    for (int r = 0; r < RB; ++r) {
      const int j = j0 + 8 * r;
      dst[r] = (col_ok && j < h.B) ? *reinterpret_cast<const uint4*>(abase + (int64_t)j * h.ld_in)
                                   : make_uint4(0u, 0u, 0u, 0u);
    }
  };
  uint4 nxt[RB];
  load_rows(nxt, warp);
  // the head's weights this thread updates: output o = t + 256 i = (class o / 64, column o % 64)
  float pw[CG], pu[CG];
#pragma unroll
  for (int i = 0; i < CG; ++i) {
    const int o = t + kHeadThreads * i, c = o / kHeadCols, n = o % kHeadCols;
    const bool v = fused && c < C && n0 + n < h.in;
    const int64_t k = rep + h.w_off + (int64_t)c * h.in + n0 + n;
    pw[i] = v ? sp.w[k] : 0.f;
    pu[i] = v && sp.u ? sp.u[k] : 0.f;
  }
  // the layer below's bias (threads 0-63, one column each)
  const bool has_prev = h.b_prev_off >= 0 && h.dz_prev;
  const bool bcol = has_prev && t < kHeadCols && n0 + t < h.in;
  const int64_t kbp = rep + h.b_prev_off + n0 + t;
  const float bpw = bcol && fused ? sp.w[kbp] : 0.f;
  const float bpu = bcol && fused && sp.u ? sp.u[kbp] : 0.f;
  // first column block: the head's bias (lane 0 of warps 0-6, classes warp, warp + 7, warp + 14)
  // and the row losses (warp 7)
  const bool first = blockIdx.x == 0;
  float hbw[3], hbu[3];
#pragma unroll
  for (int i = 0; i < 3; ++i) {
    const int c = warp + 7 * i;
    const bool v = first && fused && warp < 7 && lane == 0 && c < C;
    hbw[i] = v ? sp.w[rep + h.b_off + c] : 0.f;
    hbu[i] = v && sp.u ? sp.u[rep + h.b_off + c] : 0.f;
  }
  float rl[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int j = lane + 32 * i;
    rl[i] = first && warp == 7 && h.loss_mean && j < h.B ? h.row_loss[(int64_t)g * h.B + j] : 0.f;
  }
  for (int j = t; j < h.B; j += kHeadThreads) {
    const uint16_t* src = h.dz + ((int64_t)g * h.B + j) * h.ld_dz;
    uint16_t v[CMAX];
#pragma unroll
    for (int c = 0; c < CMAX; ++c) v[c] = c < C ? src[c] : (uint16_t)0;
#pragma unroll
    for (int c = 0; c < CMAX; ++c) dzs[j * CMAX + c] = c < C ? bf2f(v[c]) : 0.f;
  }
  __syncthreads();

  // ---- weight gradient: rows j = warp, warp + 8, ... in that order ----
  float acc[CG][8];
#pragma unroll
  for (int q = 0; q < CG; ++q)
#pragma unroll
    for (int i = 0; i < 8; ++i) acc[q][i] = 0.f;
  if (col_ok) {
    for (int j0 = warp; j0 < h.B; j0 += 8 * RB) {
      uint4 cur[RB];
#pragma unroll
      for (int r = 0; r < RB; ++r) cur[r] = nxt[r];
      if (j0 + 8 * RB < h.B) load_rows(nxt, j0 + 8 * RB);
#pragma unroll
      for (int r = 0; r < RB; ++r) {
        const int j = j0 + 8 * r;
        if (j >= h.B) break;
        float a[8];
        bf16x8_to_f32(cur[r], a);
#pragma unroll
        for (int q = 0; q < CG; ++q) {
          const float d = dzs[j * CMAX + cg * CG + q];
#pragma unroll
          for (int i = 0; i < 8; ++i) acc[q][i] = fmaf(d, a[i], acc[q][i]);
        }
      }
    }
  }
  // the layer below's bias gradient is the column sum of the bf16 data gradient the forward
  // kernel stored: thread (row group rg, 8-column chunk cc) takes rows rg, rg + 32, ...
  const int cc = t & 7, rg = t >> 3;
  const bool pcol = has_prev && n0 + cc * 8 < h.in;
  const uint16_t* pbase =
      has_prev ? h.dz_prev + (int64_t)g * h.B * h.ld_dz_prev + n0 + cc * 8 : nullptr;
  uint4 praw[PR];
#pragma unroll
  for (int r = 0; r < PR; ++r) {
    const int j = rg + 32 * r;
    praw[r] = pcol && j < h.B ? *reinterpret_cast<const uint4*>(pbase + (int64_t)j * h.ld_dz_prev)
                              : make_uint4(0u, 0u, 0u, 0u);
  }
#pragma unroll
  for (int q = 0; q < CG; ++q)
#pragma unroll
    for (int i = 0; i < 8; ++i) part[(warp * CMAX + cg * CG + q) * kHeadCols + ch * 8 + i] = acc[q][i];
  __syncthreads();
  // consecutive threads take consecutive columns of a class row; warps' partials in warp order
#pragma unroll
  for (int i = 0; i < CG; ++i) {
    const int o = t + kHeadThreads * i, c = o / kHeadCols, n = o % kHeadCols;
    if (c >= C || n0 + n >= h.in) continue;
    float s = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) s += part[(w * CMAX + c) * kHeadCols + n];
    const int64_t k = rep + h.w_off + (int64_t)c * h.in + n0 + n;
    if (!fused) {
      h.grad[k] = s;
      continue;
    }
    float w = pw[i], u = pu[i];
    update(w, u, s);
    store(k, w, u);
  }
  if (has_prev) {
    float ps[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    if (pcol) {
#pragma unroll
      for (int r = 0; r < PR; ++r) {
        float v[8];
        bf16x8_to_f32(praw[r], v);
#pragma unroll
        for (int i = 0; i < 8; ++i) ps[i] += v[i];
      }
      for (int j = rg + 32 * PR; j < h.B; j += 32) {
        float v[8];
        bf16x8_to_f32(*reinterpret_cast<const uint4*>(pbase + (int64_t)j * h.ld_dz_prev), v);
#pragma unroll
        for (int i = 0; i < 8; ++i) ps[i] += v[i];
      }
    }
    __syncthreads();  // part[] is free again
#pragma unroll
    for (int i = 0; i < 8; ++i) part[rg * kHeadCols + cc * 8 + i] = ps[i];
    __syncthreads();
    if (bcol) {
      float gb = 0.f;
#pragma unroll 8
      for (int r = 0; r < 32; ++r) gb += part[r * kHeadCols + t];  // row groups in order
      if (!fused) {
        h.grad[kbp] = gb;
      } else {
        float w = bpw, u = bpu;
        update(w, u, gb);
        store(kbp, w, u);
      }
    }
  }
  // the head's bias gradient (one warp per class, a fixed butterfly over rows) and the mean loss
  // (warp 7): the first column block of each replica
  if (first) {
    if (warp < 7) {
#pragma unroll
      for (int i = 0; i < 3; ++i) {
        const int c = warp + 7 * i;
        if (c >= C) break;
        float s = 0.f;
        for (int j = lane; j < h.B; j += 32) s += dzs[j * CMAX + c];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        if (lane == 0) {
          const int64_t k = rep + h.b_off + c;
          if (!fused) {
            h.grad[k] = s;
          } else {
            float w = hbw[i], u = hbu[i];
            update(w, u, s);
            store(k, w, u);
          }
        }
      }
    } else if (h.loss_mean) {
      float s = 0.f;
#pragma unroll
      for (int i = 0; i < 4; ++i) s += rl[i];
      for (int j = lane + 128; j < h.B; j += 32) s += h.row_loss[(int64_t)g * h.B + j];
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
    return launch_pdl(head_forward_kernel<CMAX>, grid, dim3(kHeadThreads), (size_t)h.C * h.in * 2, stream, h);
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
  return launch_pdl(head_backward_kernel<CMAX>, grid, dim3(kHeadThreads), smem, stream, h);
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
