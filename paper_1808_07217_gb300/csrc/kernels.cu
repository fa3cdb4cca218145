// Element-wise and reduction kernels of the local SGD hot path (sm_103a).
//
//  * worker mini-batch sampling (Eq. 1/2: I^k drawn from worker k's own shard) with Philox4x32-10;
//  * row gather + fp32 -> bf16 cast of the sampled inputs;
//  * fused softmax cross-entropy forward + logits gradient, least-squares loss, bias-gradient sums;
//  * the fused local momentum-SGD update over the whole flattened K x d buffer (Sec. C.3.1, A.4);
//  * the K-way model average with broadcast (Eq. 2 right; Algorithm 1's all-reduce + model update);
//  * He-normal initialisation (Sec. A.2) and small utilities.
// All of them are HBM-bound: 128-bit coalesced loads, grid-stride loops over a grid sized in
// multiples of the SM count.
#include <algorithm>

#include "../../include/lsgd.h"
#include "common.cuh"
#include "lsgd_internal.h"

namespace lsgd {

namespace {

int grid_for(int64_t work_items, int threads, int per_sm = 8) {
  int64_t blocks = (work_items + threads - 1) / threads;
  int64_t cap = (int64_t)kNumSMs * per_sm;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  return (int)blocks;
}

// ---------------------------------------------------------------------------------------------
// I^k_s[j] = k S + mulhi(word_{j mod 4}(Philox((j/4, s, k, 0), seed)), S), S = floor(N / K).
__global__ void sample_indices_kernel(int32_t* __restrict__ idx, uint32_t k0, uint32_t k1,
                                      uint32_t step, int K, int B, uint32_t S) {
  pdl_begin();
  const int groups = (B + 3) / 4;
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= K * groups) return;
  const int k = t / groups, jg = t % groups;
  const U4 r = philox4x32_10(U4{(uint32_t)jg, step, (uint32_t)k, 0u}, k0, k1);
  const uint32_t base = (uint32_t)k * S;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int j = jg * 4 + i;
    if (j < B) idx[(int64_t)k * B + j] = (int32_t)(base + mulhi32(u4_get(r, i), S));
  }
}

// ---------------------------------------------------------------------------------------------
// Reshuffling sampler.  pi_e is a keyed permutation of [0, N): a four-round balanced Feistel network
// (Luby-Rackoff) on 2h-bit values, 4^h >= N, whose round r maps (L, R) to (R, L xor F_r(R)) with
// F_r(R) = the low h bits of word 0 of Philox4x32-10((R, e, r, 2), seed); values that land outside
// [0, N) are fed through the network again (cycle walking, Black-Rogaway).  The walk from an
// i < N stays on i's cycle of the network, so it re-enters [0, N) in fewer than 4^h rounds; the
// bound only guards that fact.
__device__ __forceinline__ uint32_t feistel_pi(uint32_t i, uint32_t N, int h, uint32_t e,
                                               uint32_t k0, uint32_t k1) {
  const uint64_t mask = (1ull << h) - 1ull;
  const uint64_t dom = 1ull << (2 * h);
  uint64_t x = i;
  for (uint64_t walk = 0; walk < dom; ++walk) {
    uint64_t L = x >> h, R = x & mask;
#pragma unroll
    for (uint32_t r = 0; r < 4; ++r) {
      const U4 f = philox4x32_10(U4{(uint32_t)R, e, r, 2u}, k0, k1);
      const uint64_t nR = L ^ ((uint64_t)u4_get(f, 0) & mask);
      L = R;
      R = nR;
    }
    x = (L << h) | R;
    if (x < N) break;
  }
  return (uint32_t)x;
}

// I^k_s[j] = pi_e(k S + (t B + j) mod S): worker k's t-th step of epoch e takes the next B
// positions of its partition [k S, (k + 1) S) of the epoch's permutation.  One thread per index.
__global__ void sample_reshuffle_kernel(int32_t* __restrict__ idx, uint32_t k0, uint32_t k1,
                                        uint32_t epoch, int64_t t, int K, int B, uint32_t S,
                                        uint32_t N, int h) {
  pdl_begin();
  const int q = blockIdx.x * blockDim.x + threadIdx.x;
  if (q >= K * B) return;
  const int k = q / B, j = q % B;
  const uint32_t pos = (uint32_t)(((uint64_t)t * (uint64_t)B + (uint64_t)j) % S);
  idx[q] = (int32_t)feistel_pi((uint32_t)k * S + pos, N, h, epoch, k0, k1);
}

// ---------------------------------------------------------------------------------------------
// One CTA per gathered row; float4 loads, bf16x4 (8-byte) or float4 stores.  Each thread has
// kGatherVec of its row's float4 loads in flight at once, and the launcher sizes the CTA so that a
// row takes one such batch where it can (96 threads for D = 3072): nearly every row of a
// K x B_loc = 2048-row mini-batch is then resident at once, and the copy costs two memory round
// trips (the index, then the row) rather than one per float4 of a thread.
constexpr int kGatherVec = 8;

template <bool BF16>
__global__ void gather_rows_kernel(void* __restrict__ dst, int ld_dst, const float* __restrict__ X,
                                   int D, const int32_t* __restrict__ idx, int rows,
                                   const int32_t* __restrict__ lab_in, int32_t* __restrict__ lab_out,
                                   const float* __restrict__ t_in, float* __restrict__ t_out) {
  pdl_begin();
  const int r = blockIdx.x;
  if (r >= rows) return;
  const int64_t src_row = idx ? (int64_t)idx[r] : (int64_t)r;
  const float* src = X + src_row * D;
  if (threadIdx.x == 0) {
    if (lab_out) lab_out[r] = lab_in[src_row];
    if (t_out) t_out[r] = t_in[src_row];
  }
  const bool vec = ((D & 3) == 0) && ((ld_dst & 3) == 0);
  if (!vec) {
    for (int c = threadIdx.x; c < D; c += blockDim.x) {
      if (BF16)
        reinterpret_cast<uint16_t*>(dst)[(int64_t)r * ld_dst + c] = f2bf(src[c]);
      else
        reinterpret_cast<float*>(dst)[(int64_t)r * ld_dst + c] = src[c];
    }
    return;
  }
  const int n4 = D / 4;
  const float4* s4 = reinterpret_cast<const float4*>(src);
  for (int c0 = threadIdx.x; c0 < n4; c0 += kGatherVec * blockDim.x) {
    float4 v[kGatherVec];
#pragma unroll
    for (int i = 0; i < kGatherVec; ++i) {
      const int c = c0 + i * blockDim.x;
      if (c < n4) v[i] = __ldg(s4 + c);
    }
#pragma unroll
    for (int i = 0; i < kGatherVec; ++i) {
      const int c = c0 + i * blockDim.x;
      if (c >= n4) break;
      if (BF16) {
        uint2 o;
        o.x = (uint32_t)f2bf(v[i].x) | ((uint32_t)f2bf(v[i].y) << 16);
        o.y = (uint32_t)f2bf(v[i].z) | ((uint32_t)f2bf(v[i].w) << 16);
        reinterpret_cast<uint2*>(reinterpret_cast<uint16_t*>(dst) + (int64_t)r * ld_dst)[c] = o;
      } else {
        reinterpret_cast<float4*>(reinterpret_cast<float*>(dst) + (int64_t)r * ld_dst)[c] = v[i];
      }
    }
  }
}

// ---------------------------------------------------------------------------------------------
// Softmax cross-entropy: one CTA per group (replica), one warp per row (rows w, w + warps, ...):
// the lanes take classes lane, lane + 32, ... (coalesced loads and stores), the row's maximum and
// sum of exponentials are combined across lanes by a fixed butterfly, and the row losses by a
// fixed-shape tree in shared memory (deterministic).
template <typename TD>
__global__ void __launch_bounds__(1024) softmax_xent_kernel(
    const float* __restrict__ logits, int ld, int C, const int32_t* __restrict__ labels, int B,
    TD* __restrict__ dz, int ld_dz, float* __restrict__ loss_mean, float* __restrict__ loss_sum,
    float* __restrict__ row_out) {
  pdl_begin();
  extern __shared__ float row_loss[];  // [B]
  const int g = blockIdx.x, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nw = blockDim.x >> 5;
  const float inv_b = 1.0f / (float)B;
  if (C <= 128) {
    // up to 128 classes: a lane's (at most four) logits of RPW rows are loaded before any is used,
    // so a warp waits on memory once per RPW rows; per lane the same order as below, same bits
    constexpr int RPW = 4;
    for (int j0 = warp; j0 < B; j0 += nw * RPW) {
      float zv[RPW][4];
#pragma unroll
      for (int r = 0; r < RPW; ++r) {
        const int j = j0 + r * nw;
        const float* z = logits + ((int64_t)g * B + j) * ld;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int c = lane + 32 * i;
          zv[r][i] = (j < B && c < C) ? z[c] : -INFINITY;
        }
      }
#pragma unroll
      for (int r = 0; r < RPW; ++r) {
        const int j = j0 + r * nw;
        if (j >= B) break;  // uniform over the warp
        float mx = -INFINITY;
#pragma unroll
        for (int i = 0; i < 4; ++i)
          if (lane + 32 * i < C) mx = fmaxf(mx, zv[r][i]);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        float se = 0.f;
#pragma unroll
        for (int i = 0; i < 4; ++i)
          if (lane + 32 * i < C) se += expf(zv[r][i] - mx);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) se += __shfl_xor_sync(0xffffffffu, se, o);
        const float lse = mx + logf(se);
        const int y = labels[(int64_t)g * B + j];
        if (dz) {
          TD* dzr = dz + ((int64_t)g * B + j) * ld_dz;
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const int c = lane + 32 * i;
            if (c < C) {
              const float p = expf(zv[r][i] - lse);
              Elem<TD>::store(dzr + c, (p - (c == y ? 1.f : 0.f)) * inv_b);
            }
          }
        }
        // the label's logit: the lane that holds it
        const int yl = y & 31, yi = y >> 5;
        float zy = 0.f;
#pragma unroll
        for (int i = 0; i < 4; ++i)
          if (i == yi) zy = zv[r][i];
        zy = __shfl_sync(0xffffffffu, zy, yl);
        if (lane == 0) {
          const float l = lse - zy;
          if (row_out) row_out[(int64_t)g * B + j] = l;
          row_loss[j] = l;
        }
      }
    }
  } else {
  for (int j = warp; j < B; j += nw) {
    const float* z = logits + ((int64_t)g * B + j) * ld;
    float mx = -INFINITY;
    for (int c = lane; c < C; c += 32) mx = fmaxf(mx, z[c]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float se = 0.f;
    for (int c = lane; c < C; c += 32) se += expf(z[c] - mx);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) se += __shfl_xor_sync(0xffffffffu, se, o);
    const float lse = mx + logf(se);
    const int y = labels[(int64_t)g * B + j];
    if (dz) {
      TD* dzr = dz + ((int64_t)g * B + j) * ld_dz;
      for (int c = lane; c < C; c += 32) {
        const float p = expf(z[c] - lse);
        Elem<TD>::store(dzr + c, (p - (c == y ? 1.f : 0.f)) * inv_b);
      }
    }
    if (lane == 0) {
      const float l = lse - z[y];
      if (row_out) row_out[(int64_t)g * B + j] = l;
      row_loss[j] = l;
    }
  }
  }
  __syncthreads();
  // sum of the B row losses: a fixed tree over the rows (strides halving from the largest power
  // of two below B)
  int span = 1;
  while (span < B) span <<= 1;
  for (int st = span >> 1; st > 0; st >>= 1) {
    for (int j = threadIdx.x; j < st; j += blockDim.x)
      if (j + st < B) row_loss[j] += row_loss[j + st];
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    if (loss_mean) loss_mean[g] = row_loss[0] * inv_b;
    if (loss_sum) loss_sum[g] = row_loss[0];
  }
}

// out[g][j][n] = (the S split-K partial products part[s][g][j][n], added in split order) + bias[g][n]:
// a narrow layer's product whose reduction was split so that every SM streams.  One thread per
// output; the S loads are independent.
__global__ void split_bias_sum_kernel(const float* __restrict__ part, int S, int64_t sstride,
                                      const float* __restrict__ bias, int64_t bias_gs, int G, int B,
                                      int N, int ld, float* __restrict__ out) {
  pdl_begin();
  const int64_t total = (int64_t)G * B * N;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
       t += (int64_t)gridDim.x * blockDim.x) {
    const int n = (int)(t % N);
    const int64_t row = t / N;
    const int g = (int)(row / B);
    const int64_t off = row * ld + n;
    float v = part[off];
    for (int s = 1; s < S; ++s) v += part[(int64_t)s * sstride + off];
    out[off] = v + (bias ? bias[(int64_t)g * bias_gs + n] : 0.f);
  }
}

template <typename TD>
__global__ void lsq_loss_kernel(const float* __restrict__ z, int ld, const float* __restrict__ t,
                                int B, TD* __restrict__ dz, int ld_dz, float* __restrict__ loss_mean,
                                float* __restrict__ loss_sum, float* __restrict__ row_out) {
  pdl_begin();
  extern __shared__ float row_loss[];
  const int g = blockIdx.x;
  const float inv_b = 1.0f / (float)B;
  for (int j = threadIdx.x; j < B; j += blockDim.x) {
    const float r = z[((int64_t)g * B + j) * ld] - t[(int64_t)g * B + j];
    if (dz) Elem<TD>::store(dz + ((int64_t)g * B + j) * ld_dz, r * inv_b);
    row_loss[j] = 0.5f * r * r;
    if (row_out) row_out[(int64_t)g * B + j] = 0.5f * r * r;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float s = 0.f;
    for (int j = 0; j < B; ++j) s += row_loss[j];
    if (loss_mean) loss_mean[g] = s * inv_b;
    if (loss_sum) loss_sum[g] = s;
  }
}

// Bias gradient gb[g][o] = sum_j dz[g][j][o].  A 32 x 8 block covers 64 columns: thread (x, y) sums
// rows y, y + 8, ... of columns 2x and 2x + 1; the eight partial sums are then added in row-slice
// order through shared memory, so the result does not depend on scheduling.
template <typename TD, bool UPD>
__global__ void __launch_bounds__(256) colsum_kernel(const TD* __restrict__ dz, int ld, int B,
                                                     int out, float* __restrict__ gb, int64_t gb_gs,
                                                     SgdParams sgd) {
  pdl_begin();
  __shared__ float part[8][65];
  const int g = blockIdx.y;
  const int tx = threadIdx.x, ty = threadIdx.y;
  const int c0 = blockIdx.x * 64 + 2 * tx;
  const TD* p = dz + (int64_t)g * B * ld;
  float s0 = 0.f, s1 = 0.f;
  for (int j = ty; j < B; j += 8) {
    const TD* r = p + (int64_t)j * ld + c0;
    if (c0 < out) s0 += Elem<TD>::load(r);
    if (c0 + 1 < out) s1 += Elem<TD>::load(r + 1);
  }
  part[ty][2 * tx] = s0;
  part[ty][2 * tx + 1] = s1;
  __syncthreads();
  if (ty == 0) {
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int c = c0 + h;
      if (c >= out) continue;
      float s = 0.f;
#pragma unroll
      for (int q = 0; q < 8; ++q) s += part[q][2 * tx + h];
      const int64_t i = (int64_t)g * gb_gs + c;
      if (!UPD) {
        gb[i] = s;
      } else {
        float w = sgd.w[i], u = sgd.u ? sgd.u[i] : 0.f;
        const bool sg = sgd.sign != 0;
        if (sgd.mom == 0.f)
          sgd_elem<false, false>(w, u, s, sgd.lr, 0.f, sgd.wd, sg);
        else if (sgd.nesterov)
          sgd_elem<true, true>(w, u, s, sgd.lr, sgd.mom, sgd.wd, sg);
        else
          sgd_elem<true, false>(w, u, s, sgd.lr, sgd.mom, sgd.wd, sg);
        sgd.w[i] = w;
        if (sgd.u) sgd.u[i] = u;
        if (sgd.wb) sgd.wb[i] = f2bf(w);
      }
    }
  }
}

// ---------------------------------------------------------------------------------------------
// Fused local update (22 bytes / parameter with momentum and the bf16 shadow):
//   g' = g + lambda w (no decay where (i mod period) >= decay_end); u = m u + g';
//   w -= lr (nesterov ? g' + m u : u);   m == 0: w -= lr g'.
template <bool MOM, bool NEST, bool SHADOW>
__global__ void __launch_bounds__(256) sgd_update_kernel(
    float4* __restrict__ w, float4* __restrict__ u, const float4* __restrict__ g,
    uint2* __restrict__ wb, int64_t n4, float lr, float m, float wd, int64_t period,
    int64_t decay_end, int sgn) {
  pdl_begin();
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += stride) {
    const float4 gv = __ldcs(g + i);
    float4 wv = __ldcs(w + i);
    float lam = wd;
    if (period > 0 && ((i * 4) % period) >= decay_end) lam = 0.f;
    float4 uv = MOM ? __ldcs(u + i) : make_float4(0.f, 0.f, 0.f, 0.f);
    sgd_elem<MOM, NEST>(wv.x, uv.x, gv.x, lr, m, lam, sgn != 0);
    sgd_elem<MOM, NEST>(wv.y, uv.y, gv.y, lr, m, lam, sgn != 0);
    sgd_elem<MOM, NEST>(wv.z, uv.z, gv.z, lr, m, lam, sgn != 0);
    sgd_elem<MOM, NEST>(wv.w, uv.w, gv.w, lr, m, lam, sgn != 0);
    if (MOM) __stcs(u + i, uv);
    __stcs(w + i, wv);
    if (SHADOW) {
      uint2 o;
      o.x = (uint32_t)f2bf(wv.x) | ((uint32_t)f2bf(wv.y) << 16);
      o.y = (uint32_t)f2bf(wv.z) | ((uint32_t)f2bf(wv.w) << 16);
      __stcs(wb + i, o);
    }
  }
}

// ---------------------------------------------------------------------------------------------
// K-way average (Eq. 2 right).  A thread owns one float4 column of every replica of its group and
// walks the replicas in order with eight loads in flight (a warp's load instruction reads 512
// contiguous bytes of one replica), accumulating with two_sum_add and dividing with mean_of
// (common.cuh): the correctly rounded fp32 mean in all but hard midpoint cases, whatever K (a
// plain fp32 sum loses up to K - 1 roundings), and the mean of identical replicas is that replica.
// A column-per-thread walk keeps every load coalesced; a shuffle reduction across lanes would need
// lanes to hold different replicas of one column.
struct TwoSum4 {
  float4 s, c;
};

__device__ __forceinline__ void two_sum_add4(TwoSum4& a, const float4& v) {
  two_sum_add(a.s.x, a.c.x, v.x);
  two_sum_add(a.s.y, a.c.y, v.y);
  two_sum_add(a.s.z, a.c.z, v.z);
  two_sum_add(a.s.w, a.c.w, v.w);
}

// Average column `col` (float4 units) of K replicas spaced rs4 float4 apart, in place, and write
// its bf16 copy.
template <bool SHADOW>
__device__ __forceinline__ void average_column(float4* __restrict__ W, uint2* __restrict__ Wb, int K,
                                               int64_t rs4, int64_t col, float Kf) {
  TwoSum4 acc;
  acc.s = __ldcs(W + col);
  acc.c = make_float4(0.f, 0.f, 0.f, 0.f);
  int k = 1;
  for (; k + 8 <= K; k += 8) {
    float4 v[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) v[q] = __ldcs(W + (int64_t)(k + q) * rs4 + col);
#pragma unroll
    for (int q = 0; q < 8; ++q) two_sum_add4(acc, v[q]);
  }
  for (; k < K; ++k) two_sum_add4(acc, __ldcs(W + (int64_t)k * rs4 + col));
  float4 mean;
  if ((K & (K - 1)) == 0) {
    const float inv = 1.0f / Kf;  // exact for a power of two
    mean = make_float4(mean_of_pow2(acc.s.x, acc.c.x, Kf, inv), mean_of_pow2(acc.s.y, acc.c.y, Kf, inv),
                       mean_of_pow2(acc.s.z, acc.c.z, Kf, inv), mean_of_pow2(acc.s.w, acc.c.w, Kf, inv));
  } else {
    mean = make_float4(mean_of(acc.s.x, acc.c.x, Kf), mean_of(acc.s.y, acc.c.y, Kf),
                       mean_of(acc.s.z, acc.c.z, Kf), mean_of(acc.s.w, acc.c.w, Kf));
  }
  uint2 o;
  if (SHADOW) {
    o.x = (uint32_t)f2bf(mean.x) | ((uint32_t)f2bf(mean.y) << 16);
    o.y = (uint32_t)f2bf(mean.z) | ((uint32_t)f2bf(mean.w) << 16);
  }
  for (int kk = 0; kk < K; ++kk) {
    __stcs(W + (int64_t)kk * rs4 + col, mean);
    if (SHADOW) __stcs(Wb + (int64_t)kk * rs4 + col, o);
  }
}

template <bool SHADOW>
__global__ void __launch_bounds__(256) kway_average_kernel(float4* __restrict__ W,
                                                           uint2* __restrict__ Wb, int K,
                                                           int64_t d4) {
  pdl_begin();
  // blockIdx.y selects a group of K consecutive replicas (one group for the global average)
  W += (int64_t)blockIdx.y * K * d4;
  if (SHADOW) Wb += (int64_t)blockIdx.y * K * d4;
  const float Kf = (float)K;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t col = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; col < d4; col += stride)
    average_column<SHADOW>(W, Wb, K, d4, col, Kf);
}

// The same average restricted to a list of parameter segments of every replica (blockIdx.y =
// segment): the tensors a weight-gradient + update + average launch does not cover.
template <bool SHADOW>
__global__ void __launch_bounds__(256) kway_average_segments_kernel(float4* __restrict__ W,
                                                                    uint2* __restrict__ Wb, int K,
                                                                    int64_t rs4, AvgSegments sg) {
  pdl_begin();
  const int64_t off4 = sg.off4[blockIdx.y], n4 = sg.len4[blockIdx.y];
  const float Kf = (float)K;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += stride)
    average_column<SHADOW>(W, Wb, K, rs4, off4 + i, Kf);
}

// ---------------------------------------------------------------------------------------------
// Synchronisation variants.  L1 norms of the replicas' model differences: a block owns a chunk of
// kL1Chunk float4 columns, loads w_ref there once and walks the replicas; each replica's chunk sum
// is a fixed-shape reduction (thread, warp shuffle, warps in order), and l1_finalize_kernel adds
// the chunk sums in a fixed-shape tree, so the norms are deterministic.
constexpr int kL1Threads = 256;
constexpr int kL1PerThread = 4;
constexpr int kL1Chunk = kL1Threads * kL1PerThread;
constexpr int kL1MaxK = 1024;  // shared memory holds one value per warp and replica

template <bool EF>
__global__ void __launch_bounds__(kL1Threads) l1_partial_kernel(const float4* __restrict__ W,
                                                                const float4* __restrict__ wref,
                                                                const float4* __restrict__ E,
                                                                int K, int64_t d4, int nq,
                                                                float* __restrict__ part) {
  pdl_begin();
  extern __shared__ float red[];  // [kL1Threads / 32][K]
  const int q = blockIdx.x, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t base = (int64_t)q * kL1Chunk + threadIdx.x;
  float4 r[kL1PerThread];
  bool ok[kL1PerThread];
#pragma unroll
  for (int j = 0; j < kL1PerThread; ++j) {
    const int64_t i = base + (int64_t)j * kL1Threads;
    ok[j] = i < d4;
    r[j] = ok[j] ? wref[i] : make_float4(0.f, 0.f, 0.f, 0.f);
  }
  // replicas per batch: 32 loads in flight per thread before any is reduced
  constexpr int KB = EF ? 4 : 8;
  for (int k0 = 0; k0 < K; k0 += KB) {
    float4 v[KB][kL1PerThread], e[KB][kL1PerThread];
#pragma unroll
    for (int b = 0; b < KB; ++b)
#pragma unroll
      for (int j = 0; j < kL1PerThread; ++j) {
        const bool in = ok[j] && k0 + b < K;
        const int64_t i = (int64_t)(k0 + b) * d4 + base + (int64_t)j * kL1Threads;
        v[b][j] = in ? __ldcs(W + i) : r[j];
        e[b][j] = (EF && in) ? __ldcs(E + i) : make_float4(0.f, 0.f, 0.f, 0.f);
      }
    float s[KB];
#pragma unroll
    for (int b = 0; b < KB; ++b) {
      s[b] = 0.f;
#pragma unroll
      for (int j = 0; j < kL1PerThread; ++j)
        s[b] += fabsf(r[j].x - v[b][j].x + e[b][j].x) + fabsf(r[j].y - v[b][j].y + e[b][j].y) +
                fabsf(r[j].z - v[b][j].z + e[b][j].z) + fabsf(r[j].w - v[b][j].w + e[b][j].w);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
#pragma unroll
      for (int b = 0; b < KB; ++b) s[b] += __shfl_xor_sync(0xffffffffu, s[b], o);
    if (lane == 0)
#pragma unroll
      for (int b = 0; b < KB; ++b)
        if (k0 + b < K) red[warp * K + k0 + b] = s[b];
  }
  __syncthreads();
  for (int k = threadIdx.x; k < K; k += kL1Threads) {
    float s = 0.f;
    for (int w = 0; w < kL1Threads / 32; ++w) s += red[w * K + k];
    part[(int64_t)k * nq + q] = s;
  }
}

// p[k] = (sum of replica k's chunk sums) / d_canon: one block per replica, each thread adds a fixed
// stride of chunks in fp64, then a fixed-shape tree over the block.
__global__ void __launch_bounds__(256) l1_finalize_kernel(const float* __restrict__ part, int nq,
                                                          double d_canon, float* __restrict__ p) {
  pdl_begin();
  __shared__ double red[256];
  const int k = blockIdx.x;
  double s = 0.0;
  for (int q = threadIdx.x; q < nq; q += blockDim.x) s += part[(int64_t)k * nq + q];
  red[threadIdx.x] = s;
  __syncthreads();
  for (int w = blockDim.x / 2; w > 0; w >>= 1) {
    if (threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) p[k] = (float)(red[0] / d_canon);
}

// One thread per float4 column: sum_k sign(Delta_k) p_k, the new synchronised model, the error
// memories (EF) and the broadcast to every replica.
template <bool EF, bool SHADOW>
__global__ void __launch_bounds__(256) sign_sync_kernel(float4* __restrict__ W, uint2* __restrict__ Wb,
                                                        float4* __restrict__ wref, float4* __restrict__ E,
                                                        const float* __restrict__ p, int K,
                                                        int64_t d4) {
  pdl_begin();
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < d4; i += stride) {
    const float4 r = wref[i];
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    // one replica's contribution: sign(Delta_k) p_k, and (EF) the residual left in e^k
    auto add = [&](int k, const float4 b, const float4 e4) {
      float dv[4] = {r.x - b.x, r.y - b.y, r.z - b.z, r.w - b.w};
      if (EF) {
        dv[0] += e4.x;
        dv[1] += e4.y;
        dv[2] += e4.z;
        dv[3] += e4.w;
      }
      const float pk = p[k];
      float sp[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        sp[j] = (dv[j] > 0.f ? 1.f : (dv[j] < 0.f ? -1.f : 0.f)) * pk;
        acc[j] += sp[j];
      }
      if (EF)
        __stcs(E + (int64_t)k * d4 + i,
               make_float4(dv[0] - sp[0], dv[1] - sp[1], dv[2] - sp[2], dv[3] - sp[3]));
    };
    const float4 zero4 = make_float4(0.f, 0.f, 0.f, 0.f);
    int k = 0;
    for (; k + 4 <= K; k += 4) {
      float4 b[4], e[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        b[q] = __ldcs(W + (int64_t)(k + q) * d4 + i);
        e[q] = EF ? __ldcs(E + (int64_t)(k + q) * d4 + i) : zero4;
      }
#pragma unroll
      for (int q = 0; q < 4; ++q) add(k + q, b[q], e[q]);
    }
    for (; k < K; ++k)
      add(k, __ldcs(W + (int64_t)k * d4 + i), EF ? __ldcs(E + (int64_t)k * d4 + i) : zero4);
    const float fk = (float)K;
    const float4 nr = make_float4(r.x - acc[0] / fk, r.y - acc[1] / fk, r.z - acc[2] / fk, r.w - acc[3] / fk);
    wref[i] = nr;
    uint2 o;
    if (SHADOW) {
      o.x = (uint32_t)f2bf(nr.x) | ((uint32_t)f2bf(nr.y) << 16);
      o.y = (uint32_t)f2bf(nr.z) | ((uint32_t)f2bf(nr.w) << 16);
    }
    for (int kk = 0; kk < K; ++kk) {
      __stcs(W + (int64_t)kk * d4 + i, nr);
      if (SHADOW) __stcs(Wb + (int64_t)kk * d4 + i, o);
    }
  }
}

// Global momentum: ug = mg ug + (wref - mean_k w^k) / lr, wref -= lr ug, broadcast.  The model
// difference is accumulated as sum_k (wref - w^k) (in replica order): each term is exact or nearly
// so while w^k stays close to wref, so the difference keeps fp32 relative accuracy instead of
// inheriting the rounding error of a mean of large weights (a one-step round moves w by ~1e-3 of
// its size, where the mean's rounding alone would cost ~1e-4 relative in ug).
template <bool SHADOW>
__global__ void __launch_bounds__(256) gm_sync_kernel(float4* __restrict__ W, uint2* __restrict__ Wb,
                                                      float4* __restrict__ wref, float4* __restrict__ ug,
                                                      int K, int64_t d4, float lr, float mg) {
  pdl_begin();
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < d4; i += stride) {
    const float4 r = wref[i];
    float m[4] = {0.f, 0.f, 0.f, 0.f};
    int k = 0;
    for (; k + 8 <= K; k += 8) {
      float4 b[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) b[q] = __ldcs(W + (int64_t)(k + q) * d4 + i);
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        m[0] += r.x - b[q].x;
        m[1] += r.y - b[q].y;
        m[2] += r.z - b[q].z;
        m[3] += r.w - b[q].w;
      }
    }
    for (; k < K; ++k) {
      const float4 b = __ldcs(W + (int64_t)k * d4 + i);
      m[0] += r.x - b.x;
      m[1] += r.y - b.y;
      m[2] += r.z - b.z;
      m[3] += r.w - b.w;
    }
    float4 u = ug[i];
    const float rr[4] = {r.x, r.y, r.z, r.w};
    float uu[4] = {u.x, u.y, u.z, u.w}, nr[4];
    const float klr = (float)K * lr;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      uu[j] = fmaf(mg, uu[j], m[j] / klr);
      nr[j] = fmaf(-lr, uu[j], rr[j]);
    }
    ug[i] = make_float4(uu[0], uu[1], uu[2], uu[3]);
    const float4 n4 = make_float4(nr[0], nr[1], nr[2], nr[3]);
    wref[i] = n4;
    uint2 o;
    if (SHADOW) {
      o.x = (uint32_t)f2bf(nr[0]) | ((uint32_t)f2bf(nr[1]) << 16);
      o.y = (uint32_t)f2bf(nr[2]) | ((uint32_t)f2bf(nr[3]) << 16);
    }
    for (int kk = 0; kk < K; ++kk) {
      __stcs(W + (int64_t)kk * d4 + i, n4);
      if (SHADOW) __stcs(Wb + (int64_t)kk * d4 + i, o);
    }
  }
}

// ---------------------------------------------------------------------------------------------
// w[q] = fp32(stddev * z_q), z_q standard normal from Philox((q/4, tensor, 0, 1), seed) words
// (2p, 2p+1), p = (q/2) mod 2, by Box-Muller in fp64 (cos for even q, sin for odd q).
__global__ void init_normal_kernel(float* __restrict__ w, int64_t n, double stddev, uint32_t k0,
                                   uint32_t k1, uint32_t tensor_id) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < n; q += stride) {
    const U4 r = philox4x32_10(U4{(uint32_t)(q >> 2), tensor_id, 0u, 1u}, k0, k1);
    const int pair = (int)((q >> 1) & 1);
    const double u1 = ((double)u4_get(r, 2 * pair) + 0.5) * (1.0 / 4294967296.0);
    const double u2 = ((double)u4_get(r, 2 * pair + 1) + 0.5) * (1.0 / 4294967296.0);
    const double radius = sqrt(-2.0 * log(u1));
    const double theta = 2.0 * 3.141592653589793 * u2;
    const double z = (q & 1) ? radius * sin(theta) : radius * cos(theta);
    w[q] = (float)(stddev * z);
  }
}

__global__ void fill_kernel(float* __restrict__ w, int64_t n, float v) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) w[i] = v;
}

__global__ void broadcast_kernel(float4* __restrict__ W, int K, int64_t d4) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < d4; i += stride) {
    const float4 v = W[i];
    for (int k = 1; k < K; ++k) W[(int64_t)k * d4 + i] = v;
  }
}

__global__ void to_bf16_kernel(const float4* __restrict__ w, uint2* __restrict__ wb, int64_t n4) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += stride) {
    const float4 v = w[i];
    uint2 o;
    o.x = (uint32_t)f2bf(v.x) | ((uint32_t)f2bf(v.y) << 16);
    o.y = (uint32_t)f2bf(v.z) | ((uint32_t)f2bf(v.w) << 16);
    wb[i] = o;
  }
}

__global__ void check_finite_kernel(const float* __restrict__ w, int64_t n, int* __restrict__ flag) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  bool bad = false;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride)
    bad |= !isfinite(w[i]);
  if (__syncthreads_or(bad) && threadIdx.x == 0) atomicOr(flag, 1);
}

}  // namespace

// ---------------------------------------------------------------------------------------------
cudaError_t launch_sample_indices(int32_t* idx, uint64_t seed, int64_t step, int K, int B, int64_t N,
                                  int sampling, cudaStream_t stream) {
  if (K < 1 || B < 1 || N < K || step < 0) return cudaErrorInvalidValue;
  const int64_t S = N / K;
  if ((int64_t)K * S > 0x7fffffffLL || N > 0x7fffffffLL) return cudaErrorInvalidValue;
  if (sampling == LSGD_SAMPLE_RESHUFFLE) {
    const int64_t KB = (int64_t)K * B;
    if (KB > 0x7fffffffLL) return cudaErrorInvalidValue;
    const int64_t e = step * KB / N;            // epoch of this step
    const int64_t first = (e * N + KB - 1) / KB;  // its first step
    int h = 1;
    while ((1ll << (2 * h)) < N) ++h;
    const int threads = 128;
    const int blocks = (int)((KB + threads - 1) / threads);
    launch_pdl(sample_reshuffle_kernel, blocks, threads, 0, stream, idx, (uint32_t)seed, (uint32_t)(seed >> 32),
                                                            (uint32_t)e, step - first, K, B,
                                                            (uint32_t)S, (uint32_t)N, h);
    return cudaGetLastError();
  }
  const int groups = (B + 3) / 4;
  const int threads = 128;
  const int blocks = (int)(((int64_t)K * groups + threads - 1) / threads);
  launch_pdl(sample_indices_kernel, blocks, threads, 0, stream, idx, (uint32_t)seed, (uint32_t)(seed >> 32),
                                                        (uint32_t)step, K, B, (uint32_t)S);
  return cudaGetLastError();
}

cudaError_t launch_gather_rows(void* dst, bool dst_bf16, int ld_dst, const float* X, int D,
                               const int32_t* idx, int rows, const int32_t* labels_in,
                               int32_t* labels_out, const float* targets_in, float* targets_out,
                               cudaStream_t stream) {
  if (rows <= 0) return cudaSuccess;
  if (ld_dst < D) return cudaErrorInvalidValue;
  // one batch of kGatherVec float4 loads per thread covers the row: 96 threads for D = 3072
  const int per_row = ((D / 4 + kGatherVec - 1) / kGatherVec + 31) / 32 * 32;
  const int threads = std::min(256, std::max(32, per_row));
  if (dst_bf16)
    launch_pdl(gather_rows_kernel<true>, rows, threads, 0, stream, dst, ld_dst, X, D, idx, rows, labels_in,
                                                           labels_out, targets_in, targets_out);
  else
    launch_pdl(gather_rows_kernel<false>, rows, threads, 0, stream, dst, ld_dst, X, D, idx, rows, labels_in,
                                                            labels_out, targets_in, targets_out);
  return cudaGetLastError();
}

cudaError_t launch_softmax_xent(const float* logits, int ld, int C, const int32_t* labels, int G,
                                int B, void* dz, bool dz_bf16, int ld_dz, float* loss_mean,
                                float* loss_sum, float* row_loss, cudaStream_t stream) {
  if (G <= 0 || B <= 0) return cudaSuccess;
  if (B > 8192 || C < 1) return cudaErrorInvalidValue;
  // one warp per row, up to 32 warps (8 for at most 32 classes, where a row is one pass of a
  // warp and the block's reduction barriers would dominate); the row losses in shared memory
  const int threads = 32 * std::min(C > 32 ? 32 : 8, B);
  const size_t smem = (size_t)B * sizeof(float);
  if (dz_bf16)
    launch_pdl(softmax_xent_kernel<uint16_t>, G, threads, smem, stream,
        logits, ld, C, labels, B, reinterpret_cast<uint16_t*>(dz), ld_dz, loss_mean, loss_sum,
        row_loss);
  else
    launch_pdl(softmax_xent_kernel<float>, G, threads, smem, stream,
        logits, ld, C, labels, B, reinterpret_cast<float*>(dz), ld_dz, loss_mean, loss_sum,
        row_loss);
  return cudaGetLastError();
}

cudaError_t launch_lsq_loss(const float* z, int ld, const float* targets, int G, int B, void* dz,
                            bool dz_bf16, int ld_dz, float* loss_mean, float* loss_sum,
                            float* row_loss, cudaStream_t stream) {
  if (G <= 0 || B <= 0) return cudaSuccess;
  if (B > 8192) return cudaErrorInvalidValue;
  const size_t smem = (size_t)B * sizeof(float);
  if (dz_bf16)
    launch_pdl(lsq_loss_kernel<uint16_t>, G, 256, smem, stream, 
        z, ld, targets, B, reinterpret_cast<uint16_t*>(dz), ld_dz, loss_mean, loss_sum, row_loss);
  else
    launch_pdl(lsq_loss_kernel<float>, G, 256, smem, stream, z, ld, targets, B, reinterpret_cast<float*>(dz),
                                                     ld_dz, loss_mean, loss_sum, row_loss);
  return cudaGetLastError();
}

cudaError_t launch_split_bias_sum(const float* part, int S, int64_t sstride, const float* bias,
                                  int64_t bias_gs, int G, int B, int N, int ld, float* out,
                                  cudaStream_t stream) {
  if (G <= 0 || B <= 0 || N <= 0) return cudaSuccess;
  if (!part || !out || S < 1 || ld < N || sstride < (int64_t)G * B * ld) return cudaErrorInvalidValue;
  const int64_t total = (int64_t)G * B * N;
  const int blocks = (int)std::min<int64_t>((total + 255) / 256, 65535);
  launch_pdl(split_bias_sum_kernel, blocks, 256, 0, stream, part, S, sstride, bias, bias_gs, G, B,
             N, ld, out);
  return cudaGetLastError();
}

cudaError_t launch_colsum(const void* dz, bool dz_bf16, int ld, int G, int B, int out, float* gb,
                          int64_t gb_gs, cudaStream_t stream) {
  if (G <= 0 || out <= 0) return cudaSuccess;
  if (G > 65535) return cudaErrorInvalidValue;
  dim3 grid((out + 63) / 64, G), block(32, 8);
  const SgdParams none{};
  if (dz_bf16)
    launch_pdl(colsum_kernel<uint16_t, false>, grid, block, 0, stream, 
        reinterpret_cast<const uint16_t*>(dz), ld, B, out, gb, gb_gs, none);
  else
    launch_pdl(colsum_kernel<float, false>, grid, block, 0, stream, reinterpret_cast<const float*>(dz), ld, B,
                                                            out, gb, gb_gs, none);
  return cudaGetLastError();
}

cudaError_t launch_colsum_update(const void* dz, bool dz_bf16, int ld, int G, int B, int out,
                                 int64_t gs, const SgdParams& sgd, cudaStream_t stream) {
  if (G <= 0 || out <= 0) return cudaSuccess;
  if (G > 65535 || !sgd.w || (sgd.mom != 0.f && !sgd.u)) return cudaErrorInvalidValue;
  dim3 grid((out + 63) / 64, G), block(32, 8);
  if (dz_bf16)
    launch_pdl(colsum_kernel<uint16_t, true>, grid, block, 0, stream, reinterpret_cast<const uint16_t*>(dz),
                                                              ld, B, out, nullptr, gs, sgd);
  else
    launch_pdl(colsum_kernel<float, true>, grid, block, 0, stream, reinterpret_cast<const float*>(dz), ld, B,
                                                           out, nullptr, gs, sgd);
  return cudaGetLastError();
}

cudaError_t launch_sgd_update(float* w, float* u, const float* g, uint16_t* wb, int64_t n, float lr,
                              float momentum, int nesterov, float weight_decay, int64_t period,
                              int64_t decay_end, cudaStream_t stream, int sign_steps) {
  if (n <= 0) return cudaSuccess;
  if ((n & 3) || (period & 3) || (decay_end & 3)) return cudaErrorInvalidValue;
  const bool mom = momentum != 0.0f;
  if (mom && !u) return cudaErrorInvalidValue;
  const int64_t n4 = n / 4;
  const int threads = 256;
  const int blocks = grid_for(n4, threads, 8);
  auto W = reinterpret_cast<float4*>(w);
  auto U = reinterpret_cast<float4*>(u);
  auto G = reinterpret_cast<const float4*>(g);
  auto WB = reinterpret_cast<uint2*>(wb);
#define LSGD_UPD(M, NE, S)                                                                     \
  launch_pdl(sgd_update_kernel<M, NE, S>, blocks, threads, 0, stream, W, U, G, WB, n4, lr, momentum, \
                                                              weight_decay, period, decay_end, \
                                                              sign_steps)
  const bool sh = wb != nullptr;
  if (!mom) {
    if (sh) LSGD_UPD(false, false, true); else LSGD_UPD(false, false, false);
  } else if (nesterov) {
    if (sh) LSGD_UPD(true, true, true); else LSGD_UPD(true, true, false);
  } else {
    if (sh) LSGD_UPD(true, false, true); else LSGD_UPD(true, false, false);
  }
#undef LSGD_UPD
  return cudaGetLastError();
}

cudaError_t launch_kway_average(float* W, uint16_t* Wb, int K, int64_t d, cudaStream_t stream) {
  return launch_group_average(W, Wb, K, 1, d, stream);
}

cudaError_t launch_group_average(float* W, uint16_t* Wb, int Kp, int groups, int64_t d,
                                 cudaStream_t stream) {
  if (Kp < 1 || groups < 1 || d <= 0) return cudaSuccess;
  if ((d & 3) || groups > 65535) return cudaErrorInvalidValue;
  const int64_t d4 = d / 4;
  const int threads = 256;
  const int blocks = std::max(1, grid_for(d4, threads, 8) / groups);
  dim3 grid(blocks, groups);
  if (Wb)
    launch_pdl(kway_average_kernel<true>, grid, threads, 0, stream, reinterpret_cast<float4*>(W),
                                                            reinterpret_cast<uint2*>(Wb), Kp, d4);
  else
    launch_pdl(kway_average_kernel<false>, grid, threads, 0, stream, reinterpret_cast<float4*>(W), nullptr,
                                                             Kp, d4);
  return cudaGetLastError();
}

// Replica 0's copy of each listed segment (fp32 and bf16 shadow) to replicas 1 .. K-1
// (blockIdx.y = segment): after an average that wrote the mean to replica 0 only.
__global__ void __launch_bounds__(256) broadcast_segments_kernel(float4* __restrict__ W,
                                                                 uint2* __restrict__ Wb, int K,
                                                                 int64_t rs4, AvgSegments sg) {
  pdl_begin();
  const int64_t off4 = sg.off4[blockIdx.y], n4 = sg.len4[blockIdx.y];
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += stride) {
    const int64_t col = off4 + i;
    const float4 v = W[col];
    const uint2 b = Wb ? Wb[col] : make_uint2(0u, 0u);
    for (int k = 1; k < K; ++k) {
      __stcs(W + (int64_t)k * rs4 + col, v);
      if (Wb) __stcs(Wb + (int64_t)k * rs4 + col, b);
    }
  }
}

cudaError_t launch_broadcast_segments(float* W, uint16_t* Wb, int K, int64_t d_pad,
                                      const AvgSegments& sg, cudaStream_t stream) {
  if (K <= 1 || sg.n <= 0) return cudaSuccess;
  if ((d_pad & 3) || sg.n > kMaxAvgSegments) return cudaErrorInvalidValue;
  int64_t longest = 0;
  for (int i = 0; i < sg.n; ++i) {
    if (sg.off4[i] < 0 || sg.len4[i] < 0 || 4 * (sg.off4[i] + sg.len4[i]) > d_pad)
      return cudaErrorInvalidValue;
    longest = std::max<int64_t>(longest, sg.len4[i]);
  }
  if (longest == 0) return cudaSuccess;
  const int threads = 256;
  const int blocks = (int)std::min<int64_t>((longest + threads - 1) / threads, 2048);
  launch_pdl(broadcast_segments_kernel, dim3(blocks, sg.n), threads, 0, stream,
             reinterpret_cast<float4*>(W), reinterpret_cast<uint2*>(Wb), K, d_pad / 4, sg);
  return cudaGetLastError();
}

cudaError_t launch_average_segments(float* W, uint16_t* Wb, int K, int64_t d_pad,
                                   const AvgSegments& sg, cudaStream_t stream) {
  if (K < 1 || sg.n <= 0) return cudaSuccess;
  if ((d_pad & 3) || sg.n > kMaxAvgSegments) return cudaErrorInvalidValue;
  int64_t longest = 0;
  for (int i = 0; i < sg.n; ++i) {
    if (sg.off4[i] < 0 || sg.len4[i] < 0 || 4 * (sg.off4[i] + sg.len4[i]) > d_pad)
      return cudaErrorInvalidValue;
    longest = std::max<int64_t>(longest, sg.len4[i]);
  }
  if (longest == 0) return cudaSuccess;
  const int threads = 256;
  const int blocks = (int)std::min<int64_t>((longest + threads - 1) / threads, 1024);
  dim3 grid(blocks, sg.n);
  if (Wb)
    launch_pdl(kway_average_segments_kernel<true>, grid, threads, 0, stream,
               reinterpret_cast<float4*>(W), reinterpret_cast<uint2*>(Wb), K, d_pad / 4, sg);
  else
    launch_pdl(kway_average_segments_kernel<false>, grid, threads, 0, stream,
               reinterpret_cast<float4*>(W), nullptr, K, d_pad / 4, sg);
  return cudaGetLastError();
}

int l1_chunks(int64_t d) { return (int)((d / 4 + kL1Chunk - 1) / kL1Chunk); }

cudaError_t launch_l1_norms(const float* W, const float* wref, const float* E, int K, int64_t d,
                            int64_t d_canon, float* part, float* p, cudaStream_t stream) {
  if (K < 1 || K > kL1MaxK || d <= 0 || (d & 3)) return cudaErrorInvalidValue;
  const int nq = l1_chunks(d);
  const size_t smem = (size_t)(kL1Threads / 32) * K * sizeof(float);
  auto W4 = reinterpret_cast<const float4*>(W);
  auto R4 = reinterpret_cast<const float4*>(wref);
  auto E4 = reinterpret_cast<const float4*>(E);
  if (E)
    launch_pdl(l1_partial_kernel<true>, nq, kL1Threads, smem, stream, W4, R4, E4, K, d / 4, nq, part);
  else
    launch_pdl(l1_partial_kernel<false>, nq, kL1Threads, smem, stream, W4, R4, E4, K, d / 4, nq, part);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  launch_pdl(l1_finalize_kernel, K, 256, 0, stream, part, nq, (double)d_canon, p);
  return cudaGetLastError();
}

cudaError_t launch_sign_sync(float* W, uint16_t* Wb, float* wref, float* E, const float* p, int K,
                             int64_t d, cudaStream_t stream) {
  if (K < 1 || d <= 0 || (d & 3)) return cudaErrorInvalidValue;
  const int64_t d4 = d / 4;
  const int blocks = grid_for(d4, 256, 8);
  auto W4 = reinterpret_cast<float4*>(W);
  auto R4 = reinterpret_cast<float4*>(wref);
  auto E4 = reinterpret_cast<float4*>(E);
  auto B2 = reinterpret_cast<uint2*>(Wb);
  if (E) {
    if (Wb) launch_pdl(sign_sync_kernel<true, true>, blocks, 256, 0, stream, W4, B2, R4, E4, p, K, d4);
    else launch_pdl(sign_sync_kernel<true, false>, blocks, 256, 0, stream, W4, B2, R4, E4, p, K, d4);
  } else {
    if (Wb) launch_pdl(sign_sync_kernel<false, true>, blocks, 256, 0, stream, W4, B2, R4, E4, p, K, d4);
    else launch_pdl(sign_sync_kernel<false, false>, blocks, 256, 0, stream, W4, B2, R4, E4, p, K, d4);
  }
  return cudaGetLastError();
}

cudaError_t launch_gm_sync(float* W, uint16_t* Wb, float* wref, float* ug, int K, int64_t d,
                           float lr, float mg, cudaStream_t stream) {
  if (K < 1 || d <= 0 || (d & 3) || !(lr > 0.f)) return cudaErrorInvalidValue;
  const int64_t d4 = d / 4;
  const int blocks = grid_for(d4, 256, 8);
  auto W4 = reinterpret_cast<float4*>(W);
  auto R4 = reinterpret_cast<float4*>(wref);
  auto U4 = reinterpret_cast<float4*>(ug);
  auto B2 = reinterpret_cast<uint2*>(Wb);
  if (Wb) launch_pdl(gm_sync_kernel<true>, blocks, 256, 0, stream, W4, B2, R4, U4, K, d4, lr, mg);
  else launch_pdl(gm_sync_kernel<false>, blocks, 256, 0, stream, W4, B2, R4, U4, K, d4, lr, mg);
  return cudaGetLastError();
}

cudaError_t launch_init_normal(float* w, int64_t n, double stddev, uint64_t seed, uint32_t tensor_id,
                               cudaStream_t stream) {
  if (n <= 0) return cudaSuccess;
  init_normal_kernel<<<grid_for(n, 256, 8), 256, 0, stream>>>(w, n, stddev, (uint32_t)seed,
                                                              (uint32_t)(seed >> 32), tensor_id);
  return cudaGetLastError();
}

cudaError_t launch_fill(float* w, int64_t n, float v, cudaStream_t stream) {
  if (n <= 0) return cudaSuccess;
  fill_kernel<<<grid_for(n, 256, 8), 256, 0, stream>>>(w, n, v);
  return cudaGetLastError();
}

cudaError_t launch_broadcast(float* W, int K, int64_t d, cudaStream_t stream) {
  if (K <= 1 || d <= 0) return cudaSuccess;
  if (d & 3) return cudaErrorInvalidValue;
  broadcast_kernel<<<grid_for(d / 4, 256, 8), 256, 0, stream>>>(reinterpret_cast<float4*>(W), K,
                                                                 d / 4);
  return cudaGetLastError();
}

cudaError_t launch_to_bf16(const float* w, uint16_t* wb, int64_t n, cudaStream_t stream) {
  if (n <= 0) return cudaSuccess;
  if (n & 3) return cudaErrorInvalidValue;
  to_bf16_kernel<<<grid_for(n / 4, 256, 8), 256, 0, stream>>>(reinterpret_cast<const float4*>(w),
                                                              reinterpret_cast<uint2*>(wb), n / 4);
  return cudaGetLastError();
}

cudaError_t launch_check_finite(const float* w, int64_t n, int* flag, cudaStream_t stream) {
  if (n <= 0) return cudaSuccess;
  check_finite_kernel<<<grid_for(n, 256, 8), 256, 0, stream>>>(w, n, flag);
  return cudaGetLastError();
}

}  // namespace lsgd
