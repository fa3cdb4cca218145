// Shared device helpers of the CUDA path (never used by the oracle).
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace lsgd {

constexpr int kNumSMs = 152;  // GB300: 2 dies x 76 SMs (queried at run time where it matters)

// Philox4x32-10 (Salmon et al., SC'11): 10 rounds of the two multiply-xor lanes with the key
// bumped by the Weyl increments between rounds.  Used for the worker mini-batch indices (counter
// word 3 = 0) and the initial weights (counter word 3 = 1).
struct U4 {
  uint32_t x, y, z, w;
};

__host__ __device__ __forceinline__ uint32_t mulhi32(uint32_t a, uint32_t b) {
#ifdef __CUDA_ARCH__
  return __umulhi(a, b);
#else
  return (uint32_t)(((uint64_t)a * b) >> 32);
#endif
}

__host__ __device__ __forceinline__ U4 philox4x32_10(U4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint32_t a = 0xD2511F53u * c.x, ah = mulhi32(0xD2511F53u, c.x);
    const uint32_t b = 0xCD9E8D57u * c.z, bh = mulhi32(0xCD9E8D57u, c.z);
    c = U4{bh ^ c.y ^ k0, b, ah ^ c.w ^ k1, a};
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
  }
  return c;
}

__host__ __device__ __forceinline__ uint32_t u4_get(const U4& v, int i) {
  return i == 0 ? v.x : (i == 1 ? v.y : (i == 2 ? v.z : v.w));
}

__device__ __forceinline__ uint16_t f2bf(float f) {
  __nv_bfloat16 b = __float2bfloat16_rn(f);
  return *reinterpret_cast<uint16_t*>(&b);
}

__device__ __forceinline__ float bf2f(uint16_t u) { return __uint_as_float(((uint32_t)u) << 16); }

// One element of the local update (Sec. C.3.1 / A.4): g' = g + lam w; u = m u + g';
// w -= lr (nesterov ? g' + m u : u), or w -= lr g' without momentum; with `sgn` (the signSGD
// variant of Algorithm 4) w -= lr sign(step), sign(0) = 0.  Every kernel that updates parameters
// goes through this function, so fused and stand-alone updates agree bit for bit.
template <bool MOM, bool NEST>
__device__ __forceinline__ void sgd_elem(float& w, float& u, float g, float lr, float m, float lam,
                                         bool sgn = false) {
  const float gp = fmaf(lam, w, g);
  float st;
  if (MOM) {
    u = fmaf(m, u, gp);
    st = NEST ? fmaf(m, u, gp) : u;
  } else {
    st = gp;
  }
  if (sgn) st = st > 0.f ? 1.f : (st < 0.f ? -1.f : 0.f);
  w = fmaf(-lr, st, w);
}

// The K-way average's arithmetic (Eq. 2 right), shared by the stand-alone average and the
// weight-gradient + update + average kernel so that both give the same bits.  Replicas are added
// in order with Knuth's error-free TwoSum (s + x = t + e exactly) and the errors summed in c;
// (s + c) / K is then formed from the quotient q = s / K, the exact fma remainder s - q K and c.
// The result is the correctly rounded fp32 mean except in rare midpoint cases, whatever K.
__device__ __forceinline__ void two_sum_add(float& s, float& c, float x) {
  const float t = __fadd_rn(s, x);
  const float z = __fsub_rn(t, s);
  const float e = __fadd_rn(__fsub_rn(s, __fsub_rn(t, z)), __fsub_rn(x, z));
  s = t;
  c = __fadd_rn(c, e);
}

__device__ __forceinline__ float mean_of(float s, float c, float Kf) {
  const float q = __fdiv_rn(s, Kf);
  const float r = __fadd_rn(__fmaf_rn(-q, Kf, s), c);
  return __fadd_rn(q, __fdiv_rn(r, Kf));
}

// mean_of for K a power of two: a correctly rounded division by 2^n equals the (single-rounding)
// product with the exact reciprocal 2^-n, so this gives the same bits with two multiplies.
__device__ __forceinline__ float mean_of_pow2(float s, float c, float Kf, float invK) {
  const float q = __fmul_rn(s, invK);
  const float r = __fadd_rn(__fmaf_rn(-q, Kf, s), c);
  return __fadd_rn(q, __fmul_rn(r, invK));
}

// Programmatic dependent launch: kernels of the training step are launched so that the next one
// may be scheduled while the previous one drains.  Each such kernel first waits for the previous
// grid's completion and memory (griddepcontrol.wait) before touching global memory, and at once
// allows the next kernel to launch (its CTAs still wait here for this grid to finish).
__device__ __forceinline__ void pdl_begin() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename T>
struct Elem;
template <>
struct Elem<float> {
  __device__ __forceinline__ static float load(const float* p) { return *p; }
  __device__ __forceinline__ static void store(float* p, float v) { *p = v; }
};
template <>
struct Elem<uint16_t> {
  __device__ __forceinline__ static float load(const uint16_t* p) { return bf2f(*p); }
  __device__ __forceinline__ static void store(uint16_t* p, float v) { *p = f2bf(v); }
};

}  // namespace lsgd
