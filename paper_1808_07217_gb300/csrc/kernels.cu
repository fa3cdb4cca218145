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
// One CTA per gathered row; float4 loads, bf16x4 (8-byte) or float4 stores.
template <bool BF16>
__global__ void gather_rows_kernel(void* __restrict__ dst, int ld_dst, const float* __restrict__ X,
                                   int D, const int32_t* __restrict__ idx, int rows,
                                   const int32_t* __restrict__ lab_in, int32_t* __restrict__ lab_out,
                                   const float* __restrict__ t_in, float* __restrict__ t_out) {
  const int r = blockIdx.x;
  if (r >= rows) return;
  const int64_t src_row = idx ? (int64_t)idx[r] : (int64_t)r;
  const float* src = X + src_row * D;
  if (threadIdx.x == 0) {
    if (lab_out) lab_out[r] = lab_in[src_row];
    if (t_out) t_out[r] = t_in[src_row];
  }
  const bool vec = ((D & 3) == 0) && ((ld_dst & 3) == 0);
  if (BF16) {
    uint16_t* d = reinterpret_cast<uint16_t*>(dst) + (int64_t)r * ld_dst;
    if (vec) {
      for (int c = threadIdx.x; c < D / 4; c += blockDim.x) {
        const float4 v = __ldg(reinterpret_cast<const float4*>(src) + c);
        uint2 o;
        o.x = (uint32_t)f2bf(v.x) | ((uint32_t)f2bf(v.y) << 16);
        o.y = (uint32_t)f2bf(v.z) | ((uint32_t)f2bf(v.w) << 16);
        reinterpret_cast<uint2*>(d)[c] = o;
      }
    } else {
      for (int c = threadIdx.x; c < D; c += blockDim.x) d[c] = f2bf(src[c]);
    }
  } else {
    float* d = reinterpret_cast<float*>(dst) + (int64_t)r * ld_dst;
    if (vec) {
      for (int c = threadIdx.x; c < D / 4; c += blockDim.x)
        reinterpret_cast<float4*>(d)[c] = __ldg(reinterpret_cast<const float4*>(src) + c);
    } else {
      for (int c = threadIdx.x; c < D; c += blockDim.x) d[c] = src[c];
    }
  }
}

// ---------------------------------------------------------------------------------------------
// Softmax cross-entropy: one CTA per group (replica), one thread per row, so every row of the
// group is in flight at once.  Row losses are combined by a fixed-shape tree in shared memory
// (deterministic).
template <typename TD>
__global__ void __launch_bounds__(256) softmax_xent_kernel(
    const float* __restrict__ logits, int ld, int C, const int32_t* __restrict__ labels, int B,
    TD* __restrict__ dz, int ld_dz, float* __restrict__ loss_mean, float* __restrict__ loss_sum,
    float* __restrict__ row_out) {
  __shared__ float red[256];
  const int g = blockIdx.x;
  const float inv_b = 1.0f / (float)B;
  float acc = 0.f;
  for (int j = threadIdx.x; j < B; j += blockDim.x) {
    const float* z = logits + ((int64_t)g * B + j) * ld;
    float mx = -INFINITY;
    for (int c = 0; c < C; ++c) mx = fmaxf(mx, z[c]);
    float se = 0.f;
    for (int c = 0; c < C; ++c) se += expf(z[c] - mx);
    const float lse = mx + logf(se);
    const int y = labels[(int64_t)g * B + j];
    if (dz) {
      TD* dzr = dz + ((int64_t)g * B + j) * ld_dz;
      for (int c = 0; c < C; ++c) {
        const float p = expf(z[c] - lse);
        Elem<TD>::store(dzr + c, (p - (c == y ? 1.f : 0.f)) * inv_b);
      }
    }
    const float l = lse - z[y];
    if (row_out) row_out[(int64_t)g * B + j] = l;
    acc += l;
  }
  red[threadIdx.x] = acc;
  __syncthreads();
  for (int w = blockDim.x / 2; w > 0; w >>= 1) {
    if (threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    if (loss_mean) loss_mean[g] = red[0] * inv_b;
    if (loss_sum) loss_sum[g] = red[0];
  }
}

template <typename TD>
__global__ void lsq_loss_kernel(const float* __restrict__ z, int ld, const float* __restrict__ t,
                                int B, TD* __restrict__ dz, int ld_dz, float* __restrict__ loss_mean,
                                float* __restrict__ loss_sum, float* __restrict__ row_out) {
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
        if (sgd.mom == 0.f)
          sgd_elem<false, false>(w, u, s, sgd.lr, 0.f, sgd.wd);
        else if (sgd.nesterov)
          sgd_elem<true, true>(w, u, s, sgd.lr, sgd.mom, sgd.wd);
        else
          sgd_elem<true, false>(w, u, s, sgd.lr, sgd.mom, sgd.wd);
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
    int64_t decay_end) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += stride) {
    const float4 gv = __ldcs(g + i);
    float4 wv = __ldcs(w + i);
    float lam = wd;
    if (period > 0 && ((i * 4) % period) >= decay_end) lam = 0.f;
    float4 uv = MOM ? __ldcs(u + i) : make_float4(0.f, 0.f, 0.f, 0.f);
    sgd_elem<MOM, NEST>(wv.x, uv.x, gv.x, lr, m, lam);
    sgd_elem<MOM, NEST>(wv.y, uv.y, gv.y, lr, m, lam);
    sgd_elem<MOM, NEST>(wv.z, uv.z, gv.z, lr, m, lam);
    sgd_elem<MOM, NEST>(wv.w, uv.w, gv.w, lr, m, lam);
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
// K-way average.  A warp owns a 128-byte column block (8 float4) of every replica: lane
// (r = lane / 8, c = lane % 8) sums replicas r, r + 4, r + 8, ... of float4 column c (each load
// instruction reads four full 128-byte lines), the four partial sums are combined with two
// butterfly shuffles, and every lane writes the mean back to its replicas (fp32 and bf16).
template <bool SHADOW>
__global__ void __launch_bounds__(256) kway_average_kernel(float4* __restrict__ W,
                                                           uint2* __restrict__ Wb, int K,
                                                           int64_t d4) {
  // blockIdx.y selects a group of K consecutive replicas (one group for the global average)
  W += (int64_t)blockIdx.y * K * d4;
  if (SHADOW) Wb += (int64_t)blockIdx.y * K * d4;
  const int lane = threadIdx.x & 31;
  const int r = lane >> 3, c = lane & 7;
  const int64_t nblk = (d4 + 7) / 8;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
  const float invK = 1.0f / (float)K;
  const bool exactK = (K & (K - 1)) == 0;
  for (int64_t blk = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); blk < nblk;
       blk += warps) {
    const int64_t col = blk * 8 + c;
    const bool ok = col < d4;
    const float4 zero4 = make_float4(0.f, 0.f, 0.f, 0.f);
    float4 s = zero4;
    // Batches of eight replicas per lane (r, r + 4, ..., r + 28): all loads of a batch are issued
    // before any is summed, so up to 8 x 16 B per lane are in flight.
    for (int k = r; k < K; k += 32) {
      float4 v[8];
#pragma unroll
      for (int q = 0; q < 8; ++q)
        v[q] = (ok && k + 4 * q < K) ? __ldcs(W + (int64_t)(k + 4 * q) * d4 + col) : zero4;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        s.x += v[q].x;
        s.y += v[q].y;
        s.z += v[q].z;
        s.w += v[q].w;
      }
    }
#pragma unroll
    for (int o = 8; o <= 16; o <<= 1) {
      s.x += __shfl_xor_sync(0xffffffffu, s.x, o);
      s.y += __shfl_xor_sync(0xffffffffu, s.y, o);
      s.z += __shfl_xor_sync(0xffffffffu, s.z, o);
      s.w += __shfl_xor_sync(0xffffffffu, s.w, o);
    }
    float4 mean;
    if (exactK) {
      mean = make_float4(s.x * invK, s.y * invK, s.z * invK, s.w * invK);
    } else {
      mean = make_float4(s.x / (float)K, s.y / (float)K, s.z / (float)K, s.w / (float)K);
    }
    if (ok) {
      uint2 o;
      if (SHADOW) {
        o.x = (uint32_t)f2bf(mean.x) | ((uint32_t)f2bf(mean.y) << 16);
        o.y = (uint32_t)f2bf(mean.z) | ((uint32_t)f2bf(mean.w) << 16);
      }
      for (int kk = r; kk < K; kk += 4) {
        __stcs(W + (int64_t)kk * d4 + col, mean);
        if (SHADOW) __stcs(Wb + (int64_t)kk * d4 + col, o);
      }
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
                                  cudaStream_t stream) {
  if (K < 1 || B < 1 || N < K) return cudaErrorInvalidValue;
  const int64_t S = N / K;
  if ((int64_t)K * S > 0x7fffffffLL) return cudaErrorInvalidValue;
  const int groups = (B + 3) / 4;
  const int threads = 128;
  const int blocks = (int)(((int64_t)K * groups + threads - 1) / threads);
  sample_indices_kernel<<<blocks, threads, 0, stream>>>(idx, (uint32_t)seed, (uint32_t)(seed >> 32),
                                                        (uint32_t)step, K, B, (uint32_t)S);
  return cudaGetLastError();
}

cudaError_t launch_gather_rows(void* dst, bool dst_bf16, int ld_dst, const float* X, int D,
                               const int32_t* idx, int rows, const int32_t* labels_in,
                               int32_t* labels_out, const float* targets_in, float* targets_out,
                               cudaStream_t stream) {
  if (rows <= 0) return cudaSuccess;
  if (ld_dst < D) return cudaErrorInvalidValue;
  const int threads = D >= 1024 ? 256 : 128;
  if (dst_bf16)
    gather_rows_kernel<true><<<rows, threads, 0, stream>>>(dst, ld_dst, X, D, idx, rows, labels_in,
                                                           labels_out, targets_in, targets_out);
  else
    gather_rows_kernel<false><<<rows, threads, 0, stream>>>(dst, ld_dst, X, D, idx, rows, labels_in,
                                                            labels_out, targets_in, targets_out);
  return cudaGetLastError();
}

cudaError_t launch_softmax_xent(const float* logits, int ld, int C, const int32_t* labels, int G,
                                int B, void* dz, bool dz_bf16, int ld_dz, float* loss_mean,
                                float* loss_sum, float* row_loss, cudaStream_t stream) {
  if (G <= 0 || B <= 0) return cudaSuccess;
  if (B > 8192 || C < 1) return cudaErrorInvalidValue;
  const int threads = B >= 256 ? 256 : (B >= 128 ? 128 : (B >= 64 ? 64 : 32));
  if (dz_bf16)
    softmax_xent_kernel<uint16_t><<<G, threads, 0, stream>>>(
        logits, ld, C, labels, B, reinterpret_cast<uint16_t*>(dz), ld_dz, loss_mean, loss_sum,
        row_loss);
  else
    softmax_xent_kernel<float><<<G, threads, 0, stream>>>(
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
    lsq_loss_kernel<uint16_t><<<G, 256, smem, stream>>>(
        z, ld, targets, B, reinterpret_cast<uint16_t*>(dz), ld_dz, loss_mean, loss_sum, row_loss);
  else
    lsq_loss_kernel<float><<<G, 256, smem, stream>>>(z, ld, targets, B, reinterpret_cast<float*>(dz),
                                                     ld_dz, loss_mean, loss_sum, row_loss);
  return cudaGetLastError();
}

cudaError_t launch_colsum(const void* dz, bool dz_bf16, int ld, int G, int B, int out, float* gb,
                          int64_t gb_gs, cudaStream_t stream) {
  if (G <= 0 || out <= 0) return cudaSuccess;
  if (G > 65535) return cudaErrorInvalidValue;
  dim3 grid((out + 63) / 64, G), block(32, 8);
  const SgdParams none{};
  if (dz_bf16)
    colsum_kernel<uint16_t, false><<<grid, block, 0, stream>>>(
        reinterpret_cast<const uint16_t*>(dz), ld, B, out, gb, gb_gs, none);
  else
    colsum_kernel<float, false><<<grid, block, 0, stream>>>(reinterpret_cast<const float*>(dz), ld, B,
                                                            out, gb, gb_gs, none);
  return cudaGetLastError();
}

cudaError_t launch_colsum_update(const void* dz, bool dz_bf16, int ld, int G, int B, int out,
                                 int64_t gs, const SgdParams& sgd, cudaStream_t stream) {
  if (G <= 0 || out <= 0) return cudaSuccess;
  if (G > 65535 || !sgd.w || (sgd.mom != 0.f && !sgd.u)) return cudaErrorInvalidValue;
  dim3 grid((out + 63) / 64, G), block(32, 8);
  if (dz_bf16)
    colsum_kernel<uint16_t, true><<<grid, block, 0, stream>>>(reinterpret_cast<const uint16_t*>(dz),
                                                              ld, B, out, nullptr, gs, sgd);
  else
    colsum_kernel<float, true><<<grid, block, 0, stream>>>(reinterpret_cast<const float*>(dz), ld, B,
                                                           out, nullptr, gs, sgd);
  return cudaGetLastError();
}

cudaError_t launch_sgd_update(float* w, float* u, const float* g, uint16_t* wb, int64_t n, float lr,
                              float momentum, int nesterov, float weight_decay, int64_t period,
                              int64_t decay_end, cudaStream_t stream) {
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
  sgd_update_kernel<M, NE, S><<<blocks, threads, 0, stream>>>(W, U, G, WB, n4, lr, momentum, \
                                                              weight_decay, period, decay_end)
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
  const int64_t nblk = (d4 + 7) / 8;  // one warp per 128-byte column block
  const int threads = 256;
  const int blocks = std::max(1, grid_for(nblk * 32, threads, 8) / groups);
  dim3 grid(blocks, groups);
  if (Wb)
    kway_average_kernel<true><<<grid, threads, 0, stream>>>(reinterpret_cast<float4*>(W),
                                                            reinterpret_cast<uint2*>(Wb), Kp, d4);
  else
    kway_average_kernel<false><<<grid, threads, 0, stream>>>(reinterpret_cast<float4*>(W), nullptr,
                                                             Kp, d4);
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
