// Grouped SIMT GEMM with the dense layers' fused epilogues (sm_103a).
//
// The fp32 path (pure fp32 mode: tensor cores cannot give fp32-exact products) and the reference
// for the tcgen05 kernel's tests.  One 64 x 64 output tile per CTA, 256 threads each owning a 4 x 4
// register tile, operands staged through shared memory in 16-deep k slices.  A(m, k) and B(k, n)
// take arbitrary element strides, so one kernel serves the forward (act x W^T), data-gradient
// (dZ x W) and weight-gradient (dZ^T x act) products of Eq. 2's local gradient.
#include <algorithm>

#include "common.cuh"
#include "lsgd_internal.h"

namespace lsgd {
namespace {

constexpr int BM = 64, BN = 64, BK = 16, PAD = 4;

// splits > 1: blockIdx.z = g splits + split, k in [split kchunk, (split + 1) kchunk), and the raw
// sums go to ws (splitk_epilogue_kernel applies the epilogue).
template <typename TA, typename TB, typename TC, typename TM, int EPI>
__global__ void __launch_bounds__(256) gemm_simt_kernel(GemmArgs a, int splits, int kchunk) {
  pdl_begin();
  __shared__ __align__(16) float As[BK][BM + PAD];
  __shared__ __align__(16) float Bs[BK][BN + PAD];
  const int g = blockIdx.z / splits, split = blockIdx.z % splits;
  const int k_lo = split * kchunk, k_hi = min(a.Kd, k_lo + kchunk);
  const int m0 = blockIdx.y * BM, n0 = blockIdx.x * BN;
  const int t = threadIdx.x;
  const int tx = t & 15, ty = t >> 4;
  const TA* A = reinterpret_cast<const TA*>(a.A) + (int64_t)g * a.a_gs;
  const TB* B = reinterpret_cast<const TB*>(a.B) + (int64_t)g * a.b_gs;
  const bool a_kc = a.a_cs == 1;  // A's k index contiguous
  const bool b_nc = a.b_cs == 1;  // B's n index contiguous

  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

  for (int k0 = k_lo; k0 < k_hi; k0 += BK) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int e = t + 256 * i;
      int mm, kk;
      if (a_kc) {
        kk = e % BK;
        mm = e / BK;
      } else {
        mm = e % BM;
        kk = e / BM;
      }
      const int gm = m0 + mm, gk = k0 + kk;
      float v = 0.f;
      if (gm < a.M && gk < k_hi) v = Elem<TA>::load(A + (int64_t)gm * a.a_rs + (int64_t)gk * a.a_cs);
      As[kk][mm] = v;
      int nn;
      if (b_nc) {
        nn = e % BN;
        kk = e / BN;
      } else {
        kk = e % BK;
        nn = e / BK;
      }
      const int gn = n0 + nn, gk2 = k0 + kk;
      float vb = 0.f;
      if (gn < a.N && gk2 < k_hi)
        vb = Elem<TB>::load(B + (int64_t)gk2 * a.b_rs + (int64_t)gn * a.b_cs);
      Bs[kk][nn] = vb;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < BK; ++kk) {
      const float4 av = *reinterpret_cast<const float4*>(&As[kk][ty * 4]);
      const float4 bv = *reinterpret_cast<const float4*>(&Bs[kk][tx * 4]);
      const float ar[4] = {av.x, av.y, av.z, av.w};
      const float br[4] = {bv.x, bv.y, bv.z, bv.w};
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(ar[i], br[j], acc[i][j]);
    }
    __syncthreads();
  }

  if (splits > 1) {
    float* ws = a.ws + ((int64_t)g * splits + split) * a.M * a.N;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int m = m0 + ty * 4 + i;
      if (m >= a.M) continue;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int n = n0 + tx * 4 + j;
        if (n < a.N) ws[(int64_t)m * a.N + n] = acc[i][j];
      }
    }
    return;
  }
  TC* C = reinterpret_cast<TC*>(a.C) + (int64_t)g * a.c_gs;
  const float* bias = a.bias ? a.bias + (int64_t)g * a.bias_gs : nullptr;
  const TM* mask = a.mask ? reinterpret_cast<const TM*>(a.mask) + (int64_t)g * a.mask_gs : nullptr;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int m = m0 + ty * 4 + i;
    if (m >= a.M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + tx * 4 + j;
      if (n >= a.N) continue;
      float v = acc[i][j];
      if (EPI == EPI_BIAS || EPI == EPI_BIAS_RELU) v += bias[n];
      if (EPI == EPI_BIAS_RELU) v = fmaxf(v, 0.f);
      if (EPI == EPI_MASK) v = (Elem<TM>::load(mask + (int64_t)m * a.mask_rs + n) > 0.f) ? v : 0.f;
      Elem<TC>::store(C + (int64_t)m * a.c_rs + n, v);
    }
  }
}

// The split partial sums added in split order, then the epilogue: one thread per output.
template <typename TC, typename TM, int EPI>
__global__ void __launch_bounds__(256) splitk_epilogue_kernel(GemmArgs a, int splits) {
  pdl_begin();
  const int64_t mn = (int64_t)a.M * a.N, n_all = (int64_t)a.G * mn;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n_all; e += stride) {
    const int g = (int)(e / mn), m = (int)((e % mn) / a.N), n = (int)(e % a.N);
    const float* ws = a.ws + (int64_t)g * splits * mn + (int64_t)m * a.N + n;
    float v = 0.f;
    for (int sp = 0; sp < splits; ++sp) v += ws[sp * mn];
    if (EPI == EPI_BIAS || EPI == EPI_BIAS_RELU) v += a.bias[(int64_t)g * a.bias_gs + n];
    if (EPI == EPI_BIAS_RELU) v = fmaxf(v, 0.f);
    if (EPI == EPI_MASK)
      v = (Elem<TM>::load(reinterpret_cast<const TM*>(a.mask) + (int64_t)g * a.mask_gs +
                          (int64_t)m * a.mask_rs + n) > 0.f)
              ? v
              : 0.f;
    Elem<TC>::store(reinterpret_cast<TC*>(a.C) + (int64_t)g * a.c_gs + (int64_t)m * a.c_rs + n, v);
  }
}

template <typename TA, typename TB, typename TC, typename TM, int EPI>
cudaError_t launch_epi(const GemmArgs& a, dim3 grid, int splits, int kchunk, cudaStream_t s) {
  launch_pdl(gemm_simt_kernel<TA, TB, TC, TM, EPI>, grid, 256, 0, s, a, splits, kchunk);
  if (splits > 1) {
    const int64_t n = (int64_t)a.G * a.M * a.N;
    const int blocks = (int)std::min<int64_t>((n + 255) / 256, (int64_t)kNumSMs * 8);
    launch_pdl(splitk_epilogue_kernel<TC, TM, EPI>, blocks, 256, 0, s, a, splits);
  }
  return cudaGetLastError();
}

template <typename TA, typename TB, typename TC, typename TM>
cudaError_t dispatch_epi(const GemmArgs& a, dim3 grid, int splits, int kchunk, cudaStream_t s) {
  switch (a.epi) {
    case EPI_STORE:
      return launch_epi<TA, TB, TC, TM, EPI_STORE>(a, grid, splits, kchunk, s);
    case EPI_BIAS:
      return launch_epi<TA, TB, TC, TM, EPI_BIAS>(a, grid, splits, kchunk, s);
    case EPI_BIAS_RELU:
      return launch_epi<TA, TB, TC, TM, EPI_BIAS_RELU>(a, grid, splits, kchunk, s);
    case EPI_MASK:
      return launch_epi<TA, TB, TC, TM, EPI_MASK>(a, grid, splits, kchunk, s);
    default:
      return cudaErrorInvalidValue;
  }
}

}  // namespace

cudaError_t launch_gemm_simt(const GemmArgs& a, cudaStream_t stream) {
  if (a.M <= 0 || a.N <= 0 || a.G <= 0) return cudaSuccess;
  if (a.Kd < 0 || a.G > 65535) return cudaErrorInvalidValue;
  if ((a.epi == EPI_BIAS || a.epi == EPI_BIAS_RELU) && !a.bias) return cudaErrorInvalidValue;
  if (a.epi == EPI_MASK && !a.mask) return cudaErrorInvalidValue;
  if (a.a_bf16 != a.b_bf16) return cudaErrorInvalidValue;
  if (a.mask && a.mask_bf16 != a.a_bf16) return cudaErrorInvalidValue;
  // Few output tiles over a long reduction (a small layer's forward): cut k into splits of at
  // least 128 so that about two CTAs per SM work, as far as the workspace holds the partials.
  const int64_t tiles = (int64_t)((a.N + BN - 1) / BN) * ((a.M + BM - 1) / BM) * a.G;
  int splits = 1;
  if (a.ws && a.Kd >= 256 && tiles < kNumSMs) {
    const int64_t want = std::min<int64_t>((2 * kNumSMs + tiles - 1) / tiles, a.Kd / 128);
    const int64_t room = a.ws_floats / ((int64_t)a.G * a.M * a.N);
    splits = (int)std::max<int64_t>(1, std::min<int64_t>({want, room, (int64_t)64}));
  }
  const int kchunk = (int)(((a.Kd + splits - 1) / splits + BK - 1) / BK * BK);
  splits = kchunk > 0 ? (a.Kd + kchunk - 1) / kchunk : 1;  // every split nonempty
  if (splits < 1) splits = 1;
  dim3 grid((a.N + BN - 1) / BN, (a.M + BM - 1) / BM, a.G * splits);
  if (grid.y > 65535 || grid.z > 65535) return cudaErrorInvalidValue;
  if (a.a_bf16) {
    if (a.c_bf16)
      return dispatch_epi<uint16_t, uint16_t, uint16_t, uint16_t>(a, grid, splits, kchunk, stream);
    return dispatch_epi<uint16_t, uint16_t, float, uint16_t>(a, grid, splits, kchunk, stream);
  }
  if (a.c_bf16) return cudaErrorInvalidValue;
  return dispatch_epi<float, float, float, float>(a, grid, splits, kchunk, stream);
}

}  // namespace lsgd
