// Grouped bf16 GEMM on the 5th-generation tensor cores (tcgen05 / TMEM / TMA), sm_103a.
//
// The per-replica dense-layer products of Eq. 2's local gradient: forward act x W^T, data
// gradient dZ x W and weight gradient dZ^T x act, for K replicas at once.  Operands live in the
// replica-major buffers; each is described by one rank-3 TMA map whose outermost coordinate is the
// replica, so the CTA for (n-tile, m-tile, replica g) loads its tiles at coordinate z = g.
//
// One CTA computes a 128 x BN fp32 tile in TMEM:
//   warp 0 (one lane)  TMA producer: k-blocks of 64 bf16 (one 128-byte swizzle row) into a ring
//                      of shared-memory stages, completion signalled on the stage's mbarrier;
//   warp 1 (one lane)  MMA issuer: 4 x tcgen05.mma (M=128, N=BN, K=16) per stage, accumulate in
//                      TMEM; tcgen05.commit frees the stage and finally signals the epilogue;
//   warp 2             allocates / frees the TMEM columns;
//   warps 0-3          epilogue: tcgen05.ld of their 32 TMEM lanes (= tile rows), bias / ReLU /
//                      ReLU-mask, store to global.
// K-major operands use the canonical SWIZZLE_128B K-major layout (8-row atoms of 128 B; SBO =
// 1024 B; the k-th 16-element slice starts 32 B further); MN-major operands are loaded as
// 64-element-wide boxes stacked along MN (LBO = box stride, SBO = 1024 B; the k-th slice starts
// 16 rows = 2048 B further).  Every mbarrier wait is bounded: on expiry the kernel records an error
// flag, stops issuing, and still frees its TMEM.
//
// wgrad_update_kernel (further down) is the weight gradient fused with the local update: a
// persistent variant of the same pipeline whose epilogue streams the parameters through shared
// memory by TMA.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstdlib>
#include <mutex>
#include <type_traits>

#include "common.cuh"
#include "lsgd_internal.h"

namespace lsgd {

__device__ int g_tc_timeout = 0;

namespace {

constexpr int BM = 128;
constexpr int BK = 64;
constexpr long long kWaitCycles = 4000000000LL;  // ~2 s at 2 GHz

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

// Bounded wait on an mbarrier phase; false (and the global error flag set) on expiry.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity,
                                          long long limit_cycles = kWaitCycles) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity)) {
    if (clock64() - t0 > limit_cycles) {
      atomicExch(&g_tc_timeout, 1);
      return false;
    }
  }
  return true;
}

__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, uint64_t* bar, int x,
                                            int y, int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(x), "r"(y), "r"(z)
      : "memory");
}

__device__ __forceinline__ void tma_load_5d(void* dst, const CUtensorMap* map, uint64_t* bar, int c0,
                                            int c1, int c2, int c3, int c4) {
  asm volatile(
      "cp.async.bulk.tensor.5d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5, %6, %7}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(c0), "r"(c1), "r"(c2), "r"(c3),
      "r"(c4)
      : "memory");
}

// Shared-memory descriptor of a K-major operand whose rows are `swz` bytes (32, 64 or 128) with the
// matching swizzle: core matrices of 8 rows, SBO = 8 rows, layout code 6 / 4 / 2.
__device__ __forceinline__ uint64_t smem_desc_kmajor(uint32_t addr, uint32_t swz) {
  const uint64_t layout = swz == 128 ? 2ull : (swz == 64 ? 4ull : 6ull);
  uint64_t d = 0;
  d |= (uint64_t)((addr >> 4) & 0x3FFFu);
  d |= (uint64_t)1u << 16;  // LBO (unused by swizzled K-major layouts)
  d |= (uint64_t)(((8u * swz) >> 4) & 0x3FFFu) << 32;
  d |= 1ull << 46;
  d |= layout << 61;
  return d;
}

// An MN-major (or any) descriptor with the 32-, 64- or 128-byte swizzle given in bytes.
__device__ __forceinline__ uint64_t smem_desc_swz(uint32_t addr, uint32_t lbo, uint32_t sbo,
                                                  uint32_t swz) {
  const uint64_t layout = swz == 128 ? 2ull : (swz == 64 ? 4ull : 6ull);
  uint64_t d = 0;
  d |= (uint64_t)((addr >> 4) & 0x3FFFu);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
  d |= 1ull << 46;  // descriptor version (tcgen05)
  d |= layout << 61;
  return d;
}

__device__ __forceinline__ uint64_t smem_desc(uint32_t addr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= (uint64_t)((addr >> 4) & 0x3FFFu);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
  d |= 1ull << 46;  // descriptor version (tcgen05)
  d |= 2ull << 61;  // SWIZZLE_128B
  return d;
}

// kind::f16 instruction descriptor: fp32 accumulator, bf16 A and B, majors, N >> 3, M >> 4.
__host__ __device__ constexpr uint32_t make_idesc(int M, int N, bool a_mn, bool b_mn) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((a_mn ? 1u : 0u) << 15) | ((b_mn ? 1u : 0u) << 16) |
         ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void mma_bf16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                         uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem_d),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15},"
      " [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// Sums 16 values per lane over the 32 lanes of a warp in four halving exchanges and one final
// exchange: afterwards lane l holds the warp's sum of value l / 2 (lanes 2 j and 2 j + 1 agree).
__device__ __forceinline__ float warp_colsum16(float (&v)[16], int lane) {
#pragma unroll
  for (int w = 8; w >= 1; w >>= 1) {
    const bool up = (lane & (2 * w)) != 0;
#pragma unroll
    for (int i = 0; i < w; ++i) {
      const float send = up ? v[i] : v[i + w];
      const float keep = up ? v[i + w] : v[i];
      v[i] = keep + __shfl_xor_sync(0xffffffffu, send, 2 * w);
    }
  }
  return v[0] + __shfl_xor_sync(0xffffffffu, v[0], 1);
}

template <int BN, int STAGES>
struct Smem {
  // stage buffers first (1024-byte aligned for the 128-byte swizzle)
  uint8_t a[STAGES][BM * BK * 2];
  uint8_t b[STAGES][BN * BK * 2];
  uint64_t full[STAGES];
  uint64_t empty[STAGES];
  uint64_t accum;
  uint32_t tmem_base;
};

// ---- GEMM epilogue (one-tile and persistent kernels) ----
// One thread's 32 consecutive accumulator columns of its TMEM lane, one wait.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,"
      "%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]),
        "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]),
        "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// One thread's 64 consecutive accumulator columns of its TMEM lane: two 32-column loads, one wait.
__device__ __forceinline__ void tmem_ld64(uint32_t taddr, float (&v)[64]) {
  uint32_t r[64];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,"
      "%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%64];\n"
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,"
      "%45,%46,%47,%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63}, [%65];\n"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]),
        "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]),
        "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]), "=r"(r[32]), "=r"(r[33]), "=r"(r[34]),
        "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]), "=r"(r[40]), "=r"(r[41]),
        "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]), "=r"(r[48]),
        "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]),
        "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]),
        "=r"(r[63])
      : "r"(taddr), "r"(taddr + 32u)
      : "memory");
#pragma unroll
  for (int i = 0; i < 64; ++i) v[i] = __uint_as_float(r[i]);
}

// Sixteen consecutive outputs of one row: 32-byte stores where the row is aligned and whole,
// else element by element up to the matrix edge.
__device__ __forceinline__ void store_row16(void* C, bool c_bf16, int64_t off, int n, int N,
                                            const float (&x)[16]) {
  if (c_bf16) {
    uint16_t* out = reinterpret_cast<uint16_t*>(C) + off;
    if (n + 16 <= N && (reinterpret_cast<uintptr_t>(out) & 31) == 0) {
      uint32_t w[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) w[j] = (uint32_t)f2bf(x[2 * j]) | ((uint32_t)f2bf(x[2 * j + 1]) << 16);
      asm volatile("st.global.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(out), "r"(w[0]),
                   "r"(w[1]), "r"(w[2]), "r"(w[3]), "r"(w[4]), "r"(w[5]), "r"(w[6]), "r"(w[7])
                   : "memory");
    } else {
#pragma unroll
      for (int i = 0; i < 16; ++i)
        if (n + i < N) out[i] = f2bf(x[i]);
    }
  } else {
    float* out = reinterpret_cast<float*>(C) + off;
    if (n + 16 <= N && (reinterpret_cast<uintptr_t>(out) & 31) == 0) {
#pragma unroll
      for (int j = 0; j < 2; ++j)
        asm volatile("st.global.v8.f32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(out + 8 * j),
                     "f"(x[8 * j]), "f"(x[8 * j + 1]), "f"(x[8 * j + 2]), "f"(x[8 * j + 3]),
                     "f"(x[8 * j + 4]), "f"(x[8 * j + 5]), "f"(x[8 * j + 6]), "f"(x[8 * j + 7])
                     : "memory");
    } else {
#pragma unroll
      for (int i = 0; i < 16; ++i)
        if (n + i < N) out[i] = x[i];
    }
  }
}

// The GEMM epilogue of one 128 x BN tile for one epilogue thread: tile row et (TMEM lane et)
// leaves TMEM CW (32 or 64) columns at a time and is written straight from registers, 16 columns
// per store: C(m, n) at C + c_base + m c_rs + n, with bias (+ ReLU) or the ReLU mask of the stored
// activation applied (the row's CW mask values requested before the accumulator loads).  With
// hs_warp (bias_colsum) the stored values -- rounded to bf16 when C is bf16 -- are also summed
// over the warp's 32 rows, per column, by a fixed butterfly (rows past M add nothing); hs_warp[c]
// gets column c's partial.
template <int BN, int CW>
__device__ __forceinline__ void epilogue_rows(const TcGemmArgs& args, int et, int lane,
                                              uint32_t tmem_acc, int g, int m0, int n0,
                                              int64_t c_base, float* hs_warp) {
  static_assert(CW == 32 || CW == 64, "chunk width");
  const int m = m0 + et;
  const bool row_ok = m < args.M;
  const int epi = args.epi;
  const bool has_bias = epi == EPI_BIAS || epi == EPI_BIAS_RELU;
  const float* bias = has_bias ? args.bias + (int64_t)g * args.bias_gs : nullptr;
  const int64_t coff = c_base + (int64_t)m * args.c_rs;
  const int64_t moff = (int64_t)g * args.mask_gs + (int64_t)m * args.mask_rs;
  const uint32_t lane_base = (uint32_t)(et & ~31) << 16;
  for (int cc = 0; cc < BN; cc += CW) {
    if (n0 + cc >= args.N) break;  // uniform over the CTA
    const int nc = n0 + cc;
    // the chunk's bf16 mask words (two values each) when the row is whole and 16-byte aligned
    uint32_t mw[CW / 2];
    const uint16_t* mrow = epi == EPI_MASK && args.mask_bf16
                               ? reinterpret_cast<const uint16_t*>(args.mask) + moff + nc
                               : nullptr;
    const bool mfast = mrow && row_ok && nc + CW <= args.N &&
                       (reinterpret_cast<uintptr_t>(mrow) & 15) == 0;
    if (mfast) {
#pragma unroll
      for (int i = 0; i < CW / 8; ++i) {
        const uint4 t = __ldg(reinterpret_cast<const uint4*>(mrow) + i);
        mw[4 * i] = t.x;
        mw[4 * i + 1] = t.y;
        mw[4 * i + 2] = t.z;
        mw[4 * i + 3] = t.w;
      }
    }
    float v[CW];
    if constexpr (CW == 64)
      tmem_ld64(tmem_acc + lane_base + (uint32_t)cc, v);
    else
      tmem_ld32(tmem_acc + lane_base + (uint32_t)cc, v);
#pragma unroll
    for (int q = 0; q < CW / 16; ++q) {
      const int nb = nc + 16 * q;
      float x[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) x[i] = v[16 * q + i];
      if (has_bias) {
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const int n = nb + i;
          const float t = x[i] + (n < args.N ? __ldg(bias + n) : 0.f);
          x[i] = (epi == EPI_BIAS_RELU) ? fmaxf(t, 0.f) : t;
        }
      } else if (epi == EPI_MASK) {
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          float mv;
          if (mfast) {
            const uint32_t w = mw[8 * q + (i >> 1)];
            mv = bf2f((uint16_t)((i & 1) ? (w >> 16) : (w & 0xffffu)));
          } else {
            const int n = nb + i;
            mv = !(row_ok && n < args.N) ? 0.f
                 : args.mask_bf16 ? bf2f(reinterpret_cast<const uint16_t*>(args.mask)[moff + n])
                                  : reinterpret_cast<const float*>(args.mask)[moff + n];
          }
          x[i] = mv > 0.f ? x[i] : 0.f;
        }
      }
      if (row_ok && nb < args.N) store_row16(args.C, args.c_bf16, coff + nb, nb, args.N, x);
      if (hs_warp) {
        float t[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) t[i] = !row_ok ? 0.f : (args.c_bf16 ? bf2f(f2bf(x[i])) : x[i]);
        const float sum = warp_colsum16(t, lane);
        if (!(lane & 1)) hs_warp[cc + 16 * q + (lane >> 1)] = sum;
      }
    }
  }
}

// The bias of the layer below, for the column-sum mode: each of the 128 epilogue threads takes
// columns et + 128 i of the tile; their parameters are requested before the accumulator wait.
template <int BN>
constexpr int kBiasCols = (BN + 127) / 128;  // columns per epilogue thread

template <int BN>
__device__ __forceinline__ void bias_prefetch(const TcGemmArgs& args, int et, int g, int n0,
                                              float (&bsw)[kBiasCols<BN>],
                                              float (&bsu)[kBiasCols<BN>]) {
#pragma unroll
  for (int i = 0; i < kBiasCols<BN>; ++i) {
    const int c = 128 * i + et, n = n0 + c;
    const bool v = args.bias_colsum && args.bsgd.w && c < BN && n < args.N;
    const int64_t k = (int64_t)g * args.bias_gs + n;
    bsw[i] = v ? args.bsgd.w[k] : 0.f;
    bsu[i] = v && args.bsgd.u ? args.bsgd.u[k] : 0.f;
  }
}

// After the four warps' partials are in hs (this tile's buffer): the bias gradient of each of
// this thread's columns, (warp 0 + warp 1) + (warp 2 + warp 3), and its local update (or the
// gradient itself without bsgd.w).
template <int BN>
__device__ __forceinline__ void bias_update(const TcGemmArgs& args, int et, int g, int n0,
                                            const float (*hs)[BN], const float (&bsw)[kBiasCols<BN>],
                                            const float (&bsu)[kBiasCols<BN>]) {
#pragma unroll
  for (int i = 0; i < kBiasCols<BN>; ++i) {
    const int c = 128 * i + et, n = n0 + c;
    if (c >= BN || n >= args.N) continue;
    const float gb = __fadd_rn(__fadd_rn(hs[0][c], hs[1][c]), __fadd_rn(hs[2][c], hs[3][c]));
    const int64_t k = (int64_t)g * args.bias_gs + n;
    if (!args.bsgd.w) {
      args.bias_grad[k] = gb;
      continue;
    }
    const SgdParams& sp = args.bsgd;
    float w = bsw[i], u = bsu[i];
    const bool sg = sp.sign != 0;
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

template <int BN, int STAGES>
__global__ void __launch_bounds__(128, 1) gemm_tc_kernel(const __grid_constant__ TcGemmArgs args) {
  extern __shared__ uint8_t smem_raw[];
  Smem<BN, STAGES>& sm = *reinterpret_cast<Smem<BN, STAGES>*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int splits = args.splits > 1 ? args.splits : 1;
  const int n0 = blockIdx.x * BN, m0 = blockIdx.y * BM, g = blockIdx.z / splits;
  // implicit convolution: the tile's 128 output pixels are rows of whole images (TW = Wout) from
  // pixel m0 on, i.e. output row oy0 of image b0
  const int cv_b0 = args.conv ? m0 / (args.cv_hout * args.cv_wout) : 0;
  const int cv_oy0 = args.conv ? (m0 / args.cv_wout) % args.cv_hout : 0;
  const int split = blockIdx.z % splits;
  const int nk_all = args.conv ? (9 + 64 / args.cv_ck - 1) / (64 / args.cv_ck) : (args.Kd + BK - 1) / BK;
  const int per_split = (nk_all + splits - 1) / splits;
  const int kb_first = split * per_split;
  const int nk = min(nk_all - kb_first, per_split);  // >= 1 (the host makes every split nonempty)
  const int64_t c_base = (int64_t)g * args.c_gs + (int64_t)split * args.c_split_stride;
  const bool a_mn = args.A.mn_major, b_mn = args.B.mn_major;
  constexpr uint32_t kBytesA = BM * BK * 2, kBytesB = BN * BK * 2;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], 1);
    }
    mbar_init(&sm.accum, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 2) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(&sm.tmem_base)),
                 "r"((uint32_t)BN)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = sm.tmem_base;
  pdl_begin();  // everything above touched only shared memory and TMEM

  bool ok = true;
  if (warp == 0 && lane == 0) {
    // ---------------- TMA producer ----------------
    int issued = 0;
    for (int kb = 0; kb < nk && ok; ++kb) {
      const int s = kb % STAGES;
      const uint32_t ph = (kb / STAGES) & 1;
      if (!mbar_wait(&sm.empty[s], ph ^ 1)) {
        ok = false;
        break;
      }
      if (args.conv) {
        // 64 / Ck taps per stage; tap t: the input shifted by (kh - 1, kw - 1) (zero outside the
        // image, stride by the map's element strides) and the weights' tap-t slice [N][Ck]
        const int ck = args.cv_ck, tps = 64 / ck;
        const int t0 = (kb_first + kb) * tps, t1 = min(9, t0 + tps);
        mbar_expect_tx(&sm.full[s], (uint32_t)(t1 - t0) * (BM + BN) * ck * 2);
        for (int t = t0; t < t1; ++t) {
          const int kh = t / 3, kw = t % 3, j = t - t0;
          tma_load_5d(sm.a[s] + j * BM * ck * 2, &args.A.map, &sm.full[s], 0, kw - 1,
                      cv_oy0 * args.cv_stride + kh - 1, cv_b0, g);
          tma_load_3d(sm.b[s] + j * BN * ck * 2, &args.B.map, &sm.full[s], t * ck, n0, g);
        }
        issued = kb + 1;
        continue;
      }
      mbar_expect_tx(&sm.full[s], kBytesA + kBytesB);
      const int k0 = (kb_first + kb) * BK;
      if (!a_mn) {
        tma_load_3d(sm.a[s], &args.A.map, &sm.full[s], k0, m0, g);
      } else {
#pragma unroll
        for (int i = 0; i < BM / 64; ++i)
          tma_load_3d(sm.a[s] + i * 64 * BK * 2, &args.A.map, &sm.full[s], m0 + 64 * i, k0, g);
      }
      const int gb = args.b_shared ? 0 : g;  // identical replicas: group 0's copy for all
      if (!b_mn) {
        // K-major B: BN / box_rows boxes stacked along N (8-row swizzle atoms, rows contiguous)
        const int brows = args.B.box_rows;
        for (int i = 0; i < BN / brows; ++i)
          tma_load_3d(sm.b[s] + i * brows * BK * 2, &args.B.map, &sm.full[s], k0, n0 + i * brows, gb);
      } else {
#pragma unroll
        for (int i = 0; i < BN / 64; ++i)
          tma_load_3d(sm.b[s] + i * 64 * BK * 2, &args.B.map, &sm.full[s], n0 + 64 * i, k0, gb);
      }
      issued = kb + 1;
    }
    if (!ok) {
      // let copies already in flight land before the CTA can exit
      for (int kb = (issued > STAGES ? issued - STAGES : 0); kb < issued; ++kb)
        mbar_wait(&sm.full[kb % STAGES], (kb / STAGES) & 1);
    }
  } else if (warp == 1 && lane == 0) {
    // ---------------- MMA issuer ----------------
    constexpr uint32_t idesc_kk = make_idesc(BM, BN, false, false);
    const uint32_t idesc = idesc_kk | ((a_mn ? 1u : 0u) << 15) | ((b_mn ? 1u : 0u) << 16);
    for (int kb = 0; kb < nk; ++kb) {
      const int s = kb % STAGES;
      const uint32_t ph = (kb / STAGES) & 1;
      if (!mbar_wait(&sm.full[s], ph)) {
        ok = false;
        break;
      }
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const uint32_t a_base = smem_u32(sm.a[s]), b_base = smem_u32(sm.b[s]);
      if (args.conv) {
        // each tap's sub-tiles: rows of Ck bf16 = swz bytes; K = 16 per MMA, 32 bytes further
        const int ck = args.cv_ck, tps = 64 / ck;
        const int nt = min(9, (kb_first + kb + 1) * tps) - (kb_first + kb) * tps;
        const uint32_t swz = (uint32_t)ck * 2;
        for (int j = 0; j < nt; ++j)
          for (int kk = 0; kk < ck / 16; ++kk)
            mma_bf16(tmem, smem_desc_kmajor(a_base + j * BM * ck * 2 + kk * 32, swz),
                     smem_desc_kmajor(b_base + j * BN * ck * 2 + kk * 32, swz), idesc,
                     (kb > 0 || j > 0 || kk > 0) ? 1u : 0u);
        mma_commit(&sm.empty[s]);
        continue;
      }
#pragma unroll
      for (int kk = 0; kk < BK / 16; ++kk) {
        const uint64_t ad = a_mn ? smem_desc(a_base + kk * 2048, 64 * BK * 2, 1024)
                                 : smem_desc(a_base + kk * 32, 16, 1024);
        const uint64_t bd = b_mn ? smem_desc(b_base + kk * 2048, 64 * BK * 2, 1024)
                                 : smem_desc(b_base + kk * 32, 16, 1024);
        mma_bf16(tmem, ad, bd, idesc, (kb > 0 || kk > 0) ? 1u : 0u);
      }
      mma_commit(&sm.empty[s]);  // stage reusable once these MMAs have read it
    }
    if (ok) mma_commit(&sm.accum);  // accumulator complete
  } else if (warp >= 2 && args.epi == EPI_MASK && args.mask) {
    // warps 2-3 idle through the mainloop: they bring the tile's ReLU-mask rows (the stored
    // activation) into L1, so that the epilogue's mask loads hit L1 instead of waiting on DRAM
    // (the TMA operand loads bypass L1).  Every line prefetched starts inside the tile.
    const int esz = args.mask_bf16 ? 2 : 4;
    const int ncols = min(BN, args.N - n0);
    const int lines = (ncols * esz + 127) / 128;
    const int rows = min(BM, args.M - m0);
    const char* base = reinterpret_cast<const char*>(args.mask) +
                       ((int64_t)g * args.mask_gs + (int64_t)m0 * args.mask_rs + n0) * esz;
    for (int t = (int)threadIdx.x - 64; t < rows * lines; t += 64) {
      const int r = t / lines, l = t % lines;
      asm volatile("prefetch.global.L1 [%0];" ::"l"(base + (int64_t)r * args.mask_rs * esz + l * 128));
    }
  }
  __syncwarp();

  // ---------------- epilogue (all 4 warps) ----------------
  // Thread t writes tile row t from registers (epilogue_rows).  For the bias column sums the
  // stage buffers, free once the accumulator is complete (every MMA has read its operands), hold
  // the four warps' partials.
  float bsw[kBiasCols<BN>], bsu[kBiasCols<BN>];
  bias_prefetch<BN>(args, (int)threadIdx.x, g, n0, bsw, bsu);
  const bool have_acc = mbar_wait(&sm.accum, 0);
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  float(*hs)[BN] = reinterpret_cast<float(*)[BN]>(sm.a[0]);
  if (have_acc)
    epilogue_rows<BN, 32>(args, (int)threadIdx.x, lane, tmem, g, m0, n0, c_base,
                          args.bias_colsum ? hs[warp] : nullptr);
  if (args.bias_colsum) {
    __syncthreads();  // every thread passes it, so a wait that ran out cannot split the CTA
    if (have_acc) bias_update<BN>(args, (int)threadIdx.x, g, n0, hs, bsw, bsu);
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (warp == 2) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"((uint32_t)BN)
                 : "memory");
  }
}

// =============================================================================================
// Persistent grouped GEMM for the long products (forward and data gradient of the dense
// layers): C[g] = epilogue(A[g] B[gb]^T) over 128 x PBN output tiles.  One CTA per SM walks the
// tiles blockIdx.x, blockIdx.x + gridDim.x, ... with the replica innermost (so the CTAs that
// share a weight tile when every replica reads replica 0's, b_shared, run together and L2 serves
// it), and two TMEM accumulators let one tile's epilogue overlap the next tile's products:
//   warp 0      TMA producer: A (128 x 64) and B (PBN x 64) k-blocks into a PST-stage ring
//   warp 1      MMA issuer: tcgen05.mma (M = 128, N = PBN, K = 16), accumulator (tile & 1)
//   warp 2      TMEM allocation (2 PBN columns)
//   warps 4-7   epilogue (epilogue_rows: bias / ReLU / ReLU mask; column sums + bias
//               update): each thread writes its tile row straight from registers, each warp
//               waits for the accumulator and hands it back by itself
// 128 x 256 tiles halve the shared-memory operand bytes per MMA of the 64-wide one-tile kernel
// (whose N = 64 MMAs read as many operand bytes as they compute).
namespace pt {
constexpr int PBN = 256;
constexpr int PST = 4;  // 192 KB of operands in flight: the epilogue needs no staging tile
constexpr int THREADS = 256;
}  // namespace pt

struct PtSmem {
  uint8_t a[pt::PST][BM * BK * 2];       // 16 KB each (1024-aligned)
  uint8_t b[pt::PST][pt::PBN * BK * 2];  // 32 KB each
  float hs[2][4][pt::PBN];  // bias column sums: per tile parity, per epilogue warp
  uint64_t full[pt::PST], empty[pt::PST];
  uint64_t acc_full[2], acc_empty[2];
  uint32_t tmem_base;
  int fail;  // an epilogue warp's accumulator wait ran out (column-sum mode)
};

__global__ void __launch_bounds__(pt::THREADS, 1) gemm_pt_kernel(const __grid_constant__ TcGemmArgs args) {
  extern __shared__ uint8_t smem_raw[];
  PtSmem& sm = *reinterpret_cast<PtSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                          ~uintptr_t(1023));
  constexpr int PBN = pt::PBN, PST = pt::PST;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tiles_n = (args.N + PBN - 1) / PBN, tiles_m = (args.M + BM - 1) / BM;
  const int tiles = tiles_n * tiles_m * args.G;
  const int nk = (args.Kd + BK - 1) / BK;
  const bool a_mn = args.A.mn_major, b_mn = args.B.mn_major;
  constexpr uint32_t kBytesA = BM * BK * 2, kBytesB = PBN * BK * 2;
  // tile t: replica fastest, then m-tile, then n-tile
  auto coords = [&](int t, int& g, int& m0, int& n0) {
    g = t % args.G;
    const int r = t / args.G;
    m0 = (r % tiles_m) * BM;
    n0 = (r / tiles_m) * PBN;
  };

  if (threadIdx.x == 0) {
    for (int s = 0; s < PST; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sm.acc_full[i], 1);
      mbar_init(&sm.acc_empty[i], 4);  // one arrival per epilogue warp
    }
    sm.fail = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 2) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(&sm.tmem_base)),
                 "r"(2u * PBN)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = sm.tmem_base;
  pdl_begin();  // everything above touched only shared memory and TMEM

  if (warp == 0 && lane == 0) {
    // ---------------- TMA producer ----------------
    int it = 0;
    bool ok = true;
    for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x) {
      int g, m0, n0;
      coords(t, g, m0, n0);
      const int gb = args.b_shared ? 0 : g;  // identical replicas: replica 0's copy for all
      for (int kb = 0; kb < nk; ++kb, ++it) {
        const int s = it % PST;
        if (!mbar_wait(&sm.empty[s], ((it / PST) & 1) ^ 1)) {
          ok = false;
          break;
        }
        mbar_expect_tx(&sm.full[s], kBytesA + kBytesB);
        const int k0 = kb * BK;
        if (!a_mn) {
          tma_load_3d(sm.a[s], &args.A.map, &sm.full[s], k0, m0, g);
        } else {
#pragma unroll
          for (int i = 0; i < BM / 64; ++i)
            tma_load_3d(sm.a[s] + i * 64 * BK * 2, &args.A.map, &sm.full[s], m0 + 64 * i, k0, g);
        }
        if (!b_mn) {
          const int brows = args.B.box_rows;  // 64-row boxes stacked along N
          for (int i = 0; i < PBN / brows; ++i)
            tma_load_3d(sm.b[s] + i * brows * BK * 2, &args.B.map, &sm.full[s], k0, n0 + i * brows, gb);
        } else {
#pragma unroll
          for (int i = 0; i < PBN / 64; ++i)
            tma_load_3d(sm.b[s] + i * 64 * BK * 2, &args.B.map, &sm.full[s], n0 + 64 * i, k0, gb);
        }
      }
    }
    if (!ok) {
      for (int j = (it > PST ? it - PST : 0); j < it; ++j)
        mbar_wait(&sm.full[j % PST], (j / PST) & 1);
    }
  } else if (warp == 1 && lane == 0) {
    // ---------------- MMA issuer ----------------
    constexpr uint32_t idesc_kk = make_idesc(BM, PBN, false, false);
    const uint32_t idesc = idesc_kk | ((a_mn ? 1u : 0u) << 15) | ((b_mn ? 1u : 0u) << 16);
    int it = 0, i = 0;
    bool ok = true;
    for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x, ++i) {
      const int ab = i & 1;
      if (!mbar_wait(&sm.acc_empty[ab], ((i >> 1) & 1) ^ 1)) break;
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const uint32_t acc = tmem + (uint32_t)(ab * PBN);
      for (int kb = 0; kb < nk; ++kb, ++it) {
        const int s = it % PST;
        if (!mbar_wait(&sm.full[s], (it / PST) & 1)) {
          ok = false;
          break;
        }
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint32_t a_base = smem_u32(sm.a[s]), b_base = smem_u32(sm.b[s]);
#pragma unroll
        for (int kk = 0; kk < BK / 16; ++kk) {
          const uint64_t ad = a_mn ? smem_desc(a_base + kk * 2048, 64 * BK * 2, 1024)
                                   : smem_desc(a_base + kk * 32, 16, 1024);
          const uint64_t bd = b_mn ? smem_desc(b_base + kk * 2048, 64 * BK * 2, 1024)
                                   : smem_desc(b_base + kk * 32, 16, 1024);
          mma_bf16(acc, ad, bd, idesc, (kb > 0 || kk > 0) ? 1u : 0u);
        }
        mma_commit(&sm.empty[s]);
      }
      if (ok) mma_commit(&sm.acc_full[ab]);
    }
  } else if (warp >= 4) {
    // ---------------- epilogue ----------------
    // Each warp waits for the accumulator by itself (every lane polls; the warp goes on only if
    // all lanes saw the phase) and gives it back with one arrival.  Only the column-sum mode
    // brings the four warps together, once per tile; there a wait that ran out is shared through
    // sm.fail before that barrier, so all four leave together.
    const int et = threadIdx.x - 128, quarter = warp & 3;
    const bool colsum = args.bias_colsum;
    auto warp_wait = [&](uint64_t* bar, uint32_t parity) -> bool {
      const bool okl = mbar_wait(bar, parity);
      return __all_sync(0xffffffffu, okl);
    };
    int i = 0;
    for (int t = blockIdx.x; t < tiles; t += gridDim.x, ++i) {
      int g, m0, n0;
      coords(t, g, m0, n0);
      const int ab = i & 1;
      float bsw[kBiasCols<PBN>], bsu[kBiasCols<PBN>];
      bias_prefetch<PBN>(args, et, g, n0, bsw, bsu);
      if (args.epi == EPI_MASK && args.mask && m0 + et < args.M) {
        // this thread's row of the tile's ReLU mask (the stored activation) into L2 while the
        // tile's products run, so that the copy-out's mask loads do not each wait on DRAM
        const int esz = args.mask_bf16 ? 2 : 4;
        const int ncols = min(PBN, args.N - n0);
        const char* rowp = reinterpret_cast<const char*>(args.mask) +
                           ((int64_t)g * args.mask_gs + (int64_t)(m0 + et) * args.mask_rs + n0) * esz;
        for (int b = 0; b < ncols * esz; b += 128) asm volatile("prefetch.global.L2 [%0];" ::"l"(rowp + b));
      }
      const bool okw = warp_wait(&sm.acc_full[ab], (i >> 1) & 1);
      const uint32_t acc = tmem + (uint32_t)(ab * PBN);
      if (!colsum) {
        if (!okw) break;
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        epilogue_rows<PBN, 64>(args, et, lane, acc, g, m0, n0, (int64_t)g * args.c_gs, nullptr);
      } else {
        if (okw) {
          asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
          epilogue_rows<PBN, 64>(args, et, lane, acc, g, m0, n0, (int64_t)g * args.c_gs,
                                 sm.hs[ab][quarter]);
        } else if (lane == 0) {
          sm.fail = 1;
        }
        asm volatile("bar.sync 1, 128;" ::: "memory");
        if (*reinterpret_cast<volatile int*>(&sm.fail)) break;
        // hs[ab] is written again two tiles on, after every warp has passed the next barrier
        bias_update<PBN>(args, et, g, n0, sm.hs[ab], bsw, bsu);
      }
      asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.acc_empty[ab]);  // this warp's rows have left the accumulator
    }
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (warp == 2) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(2u * pt::PBN)
                 : "memory");
  }
}

// =============================================================================================
// Weight gradient fused with the local update: persistent, every parameter byte moved by TMA.
//
// For replica g and a 128 x 128 tile (rows m = output units, columns n = inputs) of a layer's
// weight matrix, the gradient dZ[g]^T act[g] (k = B_loc) accumulates in one of two TMEM
// accumulators while the previous tile's update runs.  The tile's parameters and momentum stream
// through a ring of shared-memory slots in 32-column chunks (128 rows x 128 B, SWIZZLE_128B), are
// updated in place, and go back to HBM by TMA stores (clipped at the matrix edge), together with
// the bf16 shadow staged in a 64-byte-swizzled buffer.  The tiles of up to two layers form one
// list (the first layer's, then the second's), so a layer's last partial wave and the launch's
// ramp are paid once for both.  One CTA per SM:
//   warp 0      operand producer: dZ / act k-blocks into a two-stage ring
//   warp 1      MMA issuer: tcgen05.mma (M = N = 128, K = 16) into accumulator (tile & 1)
//   warp 2      TMEM allocation (256 columns, 512 in averaging mode); w / u chunk producer
//   warp 3      TMA store issuer: stores each finished chunk and hands its slot back
//   warps 4-19  epilogue, four threads per tile row (TMEM lane quarter = warp % 4; warps
//               4 + 4 p .. 7 + 4 p take columns 8 p .. 8 p + 7 of each chunk): per chunk,
//               tcgen05.ld of the gradient columns, the local momentum-SGD update (weight decay,
//               heavy-ball or Nesterov momentum, Sec. A.4) on w, u in shared memory, bf16 w
//               into the slot's staging buffer.
// Each epilogue warp waits on the accumulator and chunk barriers by itself and releases the chunk
// (to the store issuer) and the accumulator (to the MMA issuer) with one arrival per warp, so the
// warps overlap one another's latencies; a wait that runs out ends that warp's loop only.
//
// Averaging mode (args.avg): the step ends with the K-way average of Eq. 2 (right), so a CTA takes
// one weight tile through all G replicas in turn (replica innermost in its tile sequence).  Each
// replica's tile gets its own gradient and local update exactly as above (u written back), and the
// updated values are summed over the replicas with the average's TwoSum in two further TMEM
// regions (s, c: columns 256-511); after the last replica the mean, divided as the average does,
// goes to replica 0's parameters and bf16 shadow -- the other replicas equal it, and the runtime
// writes their copies only when something reads them (every kernel of the next step reads
// replica 0).  Neither the per-replica updated parameters nor their shadow reach HBM.  With
// args.w_rep0 (the replicas are identical at the step's start, in either mode) each tile's
// parameters are read from replica 0.  The results equal those of this kernel in plain mode
// followed by the K-way average kernel, bit for bit.
namespace wu {
constexpr int TN = 128;                     // tile columns (= rows: BM)
constexpr int CW = 32;                      // chunk columns (fp32: one 128-byte row)
constexpr int ST = 2;                       // operand stages
constexpr int NS = 4;                       // w / u chunk slots
constexpr int SD = 2;                       // chunks whose TMA stores may be in flight (<= NS)
constexpr int EPI_WARPS = 16;               // four per TMEM lane quarter
constexpr int THREADS = 128 + 32 * EPI_WARPS;
constexpr int CPT = CW / (EPI_WARPS / 4);   // chunk columns per epilogue thread (8)
constexpr uint32_t kChunkF32 = BM * CW * 4;  // 16 KB
constexpr uint32_t kChunkB16 = BM * CW * 2;  // 8 KB
}  // namespace wu

struct WuSmem {
  uint8_t a[wu::ST][BM * BK * 2];         // 16 KB each
  uint8_t b[wu::ST][wu::TN * BK * 2];     // 16 KB each
  uint8_t w[wu::NS][wu::kChunkF32];       // 1024-aligned (SWIZZLE_128B)
  uint8_t u[wu::NS][wu::kChunkF32];
  uint8_t wb[wu::NS][wu::kChunkB16];      // bf16 staging, one per slot; 512-aligned (SWIZZLE_64B)
  uint64_t op_full[wu::ST], op_empty[wu::ST];
  uint64_t acc_full[2], acc_empty[2];
  uint64_t wu_full[wu::NS], wu_empty[wu::NS];
  uint64_t st_full[wu::NS];  // every epilogue warp has finished the slot's chunk: store it
  uint32_t tmem_base;
};

__device__ __forceinline__ void tmem_ld8(uint32_t taddr, float (&v)[8]) {
  uint32_t r[8];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];\n"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7])
      : "r"(taddr)
      : "memory");
#pragma unroll
  for (int i = 0; i < 8; ++i) v[i] = __uint_as_float(r[i]);
}

// One epilogue thread's share of a chunk: 8 gradient columns at tg and its 16-column pair region
// at tsc (s then c, 8 each), both loads in flight before one wait.
__device__ __forceinline__ void tmem_ld_g8_sc16(uint32_t tg, uint32_t tsc, float (&g)[8],
                                                float (&sc)[16]) {
  uint32_t a[8], b[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%24];\n"
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,"
      "%20,%21,%22,%23}, [%25];\n"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(a[0]), "=r"(a[1]), "=r"(a[2]), "=r"(a[3]), "=r"(a[4]), "=r"(a[5]), "=r"(a[6]),
        "=r"(a[7]), "=r"(b[0]), "=r"(b[1]), "=r"(b[2]), "=r"(b[3]), "=r"(b[4]), "=r"(b[5]),
        "=r"(b[6]), "=r"(b[7]), "=r"(b[8]), "=r"(b[9]), "=r"(b[10]), "=r"(b[11]), "=r"(b[12]),
        "=r"(b[13]), "=r"(b[14]), "=r"(b[15])
      : "r"(tg), "r"(tsc)
      : "memory");
#pragma unroll
  for (int i = 0; i < 8; ++i) g[i] = __uint_as_float(a[i]);
#pragma unroll
  for (int i = 0; i < 16; ++i) sc[i] = __uint_as_float(b[i]);
}

__device__ __forceinline__ void tmem_st16_nowait(uint32_t taddr, const float (&v)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
      "%14,%15,%16};" ::"r"(taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
      "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
      "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
      "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
      "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
      "r"(__float_as_uint(v[15]))
      : "memory");
}

// tcgen05.st has no wait of its own: tmem_wait_st before reading the columns back or freeing them.
__device__ __forceinline__ void tmem_wait_st() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tma_store_3d(const CUtensorMap* map, const void* src, int x, int y,
                                             int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%2, %3, %4}], [%1];" ::"l"(
          reinterpret_cast<uint64_t>(map)),
      "r"(smem_u32(src)), "r"(x), "r"(y), "r"(z)
      : "memory");
}

__device__ __forceinline__ int wu_chunks(int N, int n0) {
  const int left = N - n0;
  return left >= wu::TN ? wu::TN / wu::CW : (left + wu::CW - 1) / wu::CW;
}

namespace wu {
// What the epilogue does with a chunk, fixed at compile time so that the per-element code has no
// branches: PLAIN writes the updated parameters; AVG folds them into the running pair (FIRST
// starts it, LAST turns it into the mean and writes that).
enum : int { kPlain = 0, kFirst = 1, kLast = 2, kAvg = 4 };
}  // namespace wu

// The local update of four consecutive parameters under one update rule (0: no momentum,
// 1: heavy ball, 2: Nesterov) through sgd_elem, the arithmetic of every update kernel.
template <bool SG, int RULE>
__device__ __forceinline__ void sgd4_rule(float4& w, float4& u, const float4 g, const SgdParams& sp) {
  constexpr bool MOM = RULE != 0, NEST = RULE == 2;
  const float m = MOM ? sp.mom : 0.f;
  sgd_elem<MOM, NEST>(w.x, u.x, g.x, sp.lr, m, sp.wd, SG);
  sgd_elem<MOM, NEST>(w.y, u.y, g.y, sp.lr, m, sp.wd, SG);
  sgd_elem<MOM, NEST>(w.z, u.z, g.z, sp.lr, m, sp.wd, SG);
  sgd_elem<MOM, NEST>(w.w, u.w, g.w, sp.lr, m, sp.wd, SG);
}

// One epilogue thread's CPT columns of a 32-column chunk of its tile row r: the update of CPT
// parameters (w, u in the swizzled shared-memory slot rows wrow / urow), in averaging mode folded
// into the running pair (s, c) = (sc[0, CPT), sc[CPT, 2 CPT)) and, at the unit's last replica,
// replaced by the mean; wherever the parameters leave for HBM their bf16 shadow goes to brow.
// Without momentum u is neither read nor changed (its slot goes back to HBM as loaded).
template <bool SG, int RULE, int MODE>
__device__ __forceinline__ void wu_part_chunk(const float (&gv)[wu::CPT], float (&sc)[2 * wu::CPT],
                                              uint8_t* wrow, uint8_t* urow, uint8_t* brow, int part,
                                              int r, const SgdParams& sp, float Gf, float invG,
                                              bool pow2) {
  constexpr bool AVG = (MODE & wu::kAvg) != 0, FIRST = (MODE & wu::kFirst) != 0,
                 LAST = (MODE & wu::kLast) != 0;
  constexpr bool WRITE_W = !AVG || LAST;
  uint32_t packed[wu::CPT / 2];
#pragma unroll
  for (int jj = 0; jj < wu::CPT / 4; ++jj) {
    const int j = (wu::CPT / 4) * part + jj;  // float4 column group within the chunk
    const int phys = (j ^ (r & 7)) << 4;
    float4 wv = *reinterpret_cast<const float4*>(wrow + phys);
    float4 uv = RULE != 0 ? *reinterpret_cast<const float4*>(urow + phys)
                          : make_float4(0.f, 0.f, 0.f, 0.f);
    sgd4_rule<SG, RULE>(wv, uv, make_float4(gv[4 * jj], gv[4 * jj + 1], gv[4 * jj + 2], gv[4 * jj + 3]),
                        sp);
    if (RULE != 0) *reinterpret_cast<float4*>(urow + phys) = uv;
    if (AVG) {
      float* sv = sc + 4 * jj;            // s of these four columns
      float* cv = sc + wu::CPT + 4 * jj;  // c of these four columns
      const float wn[4] = {wv.x, wv.y, wv.z, wv.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        if (FIRST) {
          sv[e] = wn[e];
          cv[e] = 0.f;
        } else {
          two_sum_add(sv[e], cv[e], wn[e]);
        }
      }
      if (LAST) {
        float m[4];
        if (pow2) {
#pragma unroll
          for (int e = 0; e < 4; ++e) m[e] = mean_of_pow2(sv[e], cv[e], Gf, invG);
        } else {
#pragma unroll
          for (int e = 0; e < 4; ++e) m[e] = mean_of(sv[e], cv[e], Gf);
        }
        wv = make_float4(m[0], m[1], m[2], m[3]);
      }
    }
    if (WRITE_W) {
      *reinterpret_cast<float4*>(wrow + phys) = wv;
      packed[2 * jj] = (uint32_t)f2bf(wv.x) | ((uint32_t)f2bf(wv.y) << 16);
      packed[2 * jj + 1] = (uint32_t)f2bf(wv.z) | ((uint32_t)f2bf(wv.w) << 16);
    }
  }
  if (WRITE_W) {
#pragma unroll
    for (int hh = 0; hh < wu::CPT / 8; ++hh) {
      const int h = (wu::CPT / 8) * part + hh;  // 16-byte unit of the 64-byte bf16 row
      *reinterpret_cast<uint4*>(brow + ((h ^ ((r >> 1) & 3)) << 4)) =
          make_uint4(packed[4 * hh], packed[4 * hh + 1], packed[4 * hh + 2], packed[4 * hh + 3]);
    }
  }
}

__global__ void __launch_bounds__(wu::THREADS, 1) wgrad_update_kernel(
    const __grid_constant__ WgradUpdateArgs args) {
  extern __shared__ uint8_t smem_raw[];
  WuSmem& sm = *reinterpret_cast<WuSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                          ~uintptr_t(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // the layers' tiles one layer after another (operand layouts are the same in all): layer l's
  // tiles follow uc_l tile positions (uc_l G tiles) of the layers before it (scalars, so that
  // nothing needs local memory)
  static_assert(kWgradMaxLayers == 3, "the bookkeeping below names three layers");
  const int tn0 = (args.L[0].N + wu::TN - 1) / wu::TN;
  const int tn1 = args.nl > 1 ? (args.L[1].N + wu::TN - 1) / wu::TN : 0;
  const int tn2 = args.nl > 2 ? (args.L[2].N + wu::TN - 1) / wu::TN : 0;
  const int uc1 = tn0 * ((args.L[0].M + BM - 1) / BM);
  const int uc2 = uc1 + (args.nl > 1 ? tn1 * ((args.L[1].M + BM - 1) / BM) : 0);
  const int uc3 = uc2 + (args.nl > 2 ? tn2 * ((args.L[2].M + BM - 1) / BM) : 0);
  const int tiles = uc3 * args.G;
  const int nk = (args.Kd + BK - 1) / BK;
  const bool a_mn = args.L[0].A.mn_major, b_mn = args.L[0].B.mn_major;
  const bool has_u = args.sgd.u != nullptr;
  const bool avg = args.avg != 0;
  constexpr uint32_t kBytesA = BM * BK * 2, kBytesB = wu::TN * BK * 2;
  // This CTA's tile sequence: units blockIdx.x, blockIdx.x + gridDim.x, ...; a unit is one tile,
  // or one tile position of a layer taken through all G replicas -- in averaging mode, and
  // whenever every replica reads replica 0's parameters (w_rep0): then replica 0's tile comes
  // last, so that no replica reads it after it has been updated.
  const bool by_unit = avg || args.w_rep0;
  const int units = by_unit ? uc3 : tiles;
  const int per_unit = by_unit ? args.G : 1;
  const int my_count =
      (int)blockIdx.x < units ? ((units - 1 - (int)blockIdx.x) / (int)gridDim.x + 1) * per_unit : 0;
  const uint32_t tmem_cols = avg ? 4u * wu::TN : 2u * wu::TN;

  if (threadIdx.x == 0) {
    for (int i = 0; i < wu::ST; ++i) {
      mbar_init(&sm.op_full[i], 1);
      mbar_init(&sm.op_empty[i], 1);
    }
    // the epilogue warps release the accumulator and the chunk slots one arrival per warp
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sm.acc_full[i], 1);
      mbar_init(&sm.acc_empty[i], wu::EPI_WARPS);
    }
    for (int i = 0; i < wu::NS; ++i) {
      mbar_init(&sm.wu_full[i], 1);
      mbar_init(&sm.wu_empty[i], 1);
      mbar_init(&sm.st_full[i], wu::EPI_WARPS);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 2) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(&sm.tmem_base)),
                 "r"(tmem_cols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = sm.tmem_base;
  pdl_begin();  // everything above touched only shared memory and TMEM

  // tile position x (< uc3) -> its layer l, the position within the layer and the layer's
  // column-tile count
  auto locate = [&](int x, int& l, int& r, int& tnl) {
    l = (x >= uc1 ? 1 : 0) + (x >= uc2 ? 1 : 0);
    r = x - (l == 0 ? 0 : (l == 1 ? uc1 : uc2));
    tnl = l == 0 ? tn0 : (l == 1 ? tn1 : tn2);
  };
  auto tile_coords = [&](int t, const WgradUpdateLayer*& ly, int& g, int& m0, int& n0) {
    // layer by layer, each layer's tiles replica by replica
    const int l0 = (t >= uc1 * args.G ? 1 : 0) + (t >= uc2 * args.G ? 1 : 0);
    const int base = l0 == 0 ? 0 : (l0 == 1 ? uc1 : uc2);
    const int per_g = (l0 == 0 ? uc1 : (l0 == 1 ? uc2 : uc3)) - base;
    t -= base * args.G;
    g = t / per_g;
    int l, r, tnl;
    locate(base + t % per_g, l, r, tnl);
    ly = &args.L[l];
    m0 = (r / tnl) * BM;
    n0 = (r % tnl) * wu::TN;
  };
  // the j-th tile of this CTA's sequence; gi = its replica's position within the unit
  auto tile_at = [&](int j, const WgradUpdateLayer*& ly, int& g, int& m0, int& n0, int& gi) {
    const int u = (int)blockIdx.x + (j / per_unit) * (int)gridDim.x;
    gi = j % per_unit;
    if (!by_unit) {
      tile_coords(u, ly, g, m0, n0);
      return;
    }
    int l, r, tnl;
    locate(u, l, r, tnl);
    ly = &args.L[l];
    m0 = (r / tnl) * BM;
    n0 = (r % tnl) * wu::TN;
    // averaging: replicas in order (the average's summation order); else replica 0 last
    g = avg ? gi : (gi + 1) % args.G;
  };

  if (warp == 0 && lane == 0) {
    // ---------------- operand producer ----------------
    int it = 0;
    bool ok = true;
    for (int j = 0; j < my_count && ok; ++j) {
      const WgradUpdateLayer* ly;
      int g, m0, n0, gi;
      tile_at(j, ly, g, m0, n0, gi);
      for (int kb = 0; kb < nk; ++kb, ++it) {
        const int s = it % wu::ST;
        if (!mbar_wait(&sm.op_empty[s], ((it / wu::ST) & 1) ^ 1)) {
          ok = false;
          break;
        }
        mbar_expect_tx(&sm.op_full[s], kBytesA + kBytesB);
        const int k0 = kb * BK;
        if (!a_mn) {
          tma_load_3d(sm.a[s], &ly->A.map, &sm.op_full[s], k0, m0, g);
        } else {
#pragma unroll
          for (int i = 0; i < BM / 64; ++i)
            tma_load_3d(sm.a[s] + i * 64 * BK * 2, &ly->A.map, &sm.op_full[s], m0 + 64 * i, k0, g);
        }
        if (!b_mn) {
          tma_load_3d(sm.b[s], &ly->B.map, &sm.op_full[s], k0, n0, g);
        } else {
#pragma unroll
          for (int i = 0; i < wu::TN / 64; ++i)
            tma_load_3d(sm.b[s] + i * 64 * BK * 2, &ly->B.map, &sm.op_full[s], n0 + 64 * i, k0, g);
        }
      }
    }
    if (!ok) {
      // let copies in flight land before the CTA can exit
      for (int j = (it > wu::ST ? it - wu::ST : 0); j < it; ++j)
        mbar_wait(&sm.op_full[j % wu::ST], (j / wu::ST) & 1);
    }
  } else if (warp == 1 && lane == 0) {
    // ---------------- MMA issuer ----------------
    const uint32_t idesc = make_idesc(BM, wu::TN, a_mn, b_mn);
    int it = 0, i = 0;
    bool ok = true;
    for (; i < my_count && ok; ++i) {
      const int ab = i & 1;
      if (!mbar_wait(&sm.acc_empty[ab], ((i >> 1) & 1) ^ 1)) break;
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const uint32_t acc = tmem + (uint32_t)(ab * wu::TN);
      for (int kb = 0; kb < nk; ++kb, ++it) {
        const int s = it % wu::ST;
        if (!mbar_wait(&sm.op_full[s], (it / wu::ST) & 1)) {
          ok = false;
          break;
        }
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint32_t a_base = smem_u32(sm.a[s]), b_base = smem_u32(sm.b[s]);
#pragma unroll
        for (int kk = 0; kk < BK / 16; ++kk) {
          const uint64_t ad = a_mn ? smem_desc(a_base + kk * 2048, 64 * BK * 2, 1024)
                                   : smem_desc(a_base + kk * 32, 16, 1024);
          const uint64_t bd = b_mn ? smem_desc(b_base + kk * 2048, 64 * BK * 2, 1024)
                                   : smem_desc(b_base + kk * 32, 16, 1024);
          mma_bf16(acc, ad, bd, idesc, (kb > 0 || kk > 0) ? 1u : 0u);
        }
        mma_commit(&sm.op_empty[s]);
      }
      if (ok) mma_commit(&sm.acc_full[ab]);
    }
  } else if (warp == 2 && lane == 0) {
    // ---------------- w / u chunk producer ----------------
    int q = 0;
    bool ok = true;
    const uint32_t bytes = wu::kChunkF32 * (has_u ? 2u : 1u);
    for (int j = 0; j < my_count && ok; ++j) {
      const WgradUpdateLayer* ly;
      int g, m0, n0, gi;
      tile_at(j, ly, g, m0, n0, gi);
      const int gw = args.w_rep0 ? 0 : g;  // identical replicas: read replica 0's
      const int nc = wu_chunks(ly->N, n0);
      for (int c = 0; c < nc; ++c, ++q) {
        const int sl = q % wu::NS;
        if (!mbar_wait(&sm.wu_empty[sl], ((q / wu::NS) & 1) ^ 1)) {
          ok = false;
          break;
        }
        mbar_expect_tx(&sm.wu_full[sl], bytes);
        tma_load_3d(sm.w[sl], &ly->wmap, &sm.wu_full[sl], n0 + c * wu::CW, m0, gw);
        if (has_u) tma_load_3d(sm.u[sl], &ly->umap, &sm.wu_full[sl], n0 + c * wu::CW, m0, g);
      }
    }
    if (!ok) {
      for (int j = (q > wu::NS ? q - wu::NS : 0); j < q; ++j)
        mbar_wait(&sm.wu_full[j % wu::NS], (j / wu::NS) & 1);
    }
  } else if (warp == 3 && lane == 0) {
    // ---------------- store issuer ----------------
    // Each finished chunk leaves by TMA stores (u; the updated w and its bf16 shadow, or in
    // averaging mode at the unit's last replica the mean to replica 0); once they have read the
    // slot it goes back to the w / u producer.  Issuing stores here keeps their cost (a few
    // hundred cycles each) off the epilogue threads.
    int q = 0;
    bool ok = true;
    for (int j = 0; j < my_count && ok; ++j) {
      const WgradUpdateLayer* ly;
      int g, m0, n0, gi;
      tile_at(j, ly, g, m0, n0, gi);
      const bool last = gi == per_unit - 1;
      const int nc = wu_chunks(ly->N, n0);
      for (int c = 0; c < nc; ++c, ++q) {
        const int sl = q % wu::NS;
        if (!mbar_wait(&sm.st_full[sl], (q / wu::NS) & 1)) {
          ok = false;
          break;
        }
        const int x = n0 + c * wu::CW;
        if (has_u) tma_store_3d(&ly->umap, sm.u[sl], x, m0, g);
        if (!avg) {
          tma_store_3d(&ly->wmap, sm.w[sl], x, m0, g);
          if (args.sgd.wb) tma_store_3d(&ly->wbmap, sm.wb[sl], x, m0, g);
        } else if (last) {
          // the mean goes to replica 0 only; the runtime copies it to the other replicas when
          // something needs them (every consumer of the next step reads replica 0)
          tma_store_3d(&ly->wmap, sm.w[sl], x, m0, 0);
          if (args.sgd.wb) tma_store_3d(&ly->wbmap, sm.wb[sl], x, m0, 0);
        }
        asm volatile("cp.async.bulk.commit_group;" ::: "memory");
        // SD chunks' store groups in flight: once at most SD - 1 are still reading shared
        // memory, the oldest one's slot goes back to the w / u producer
        asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(wu::SD - 1) : "memory");
        if (q >= wu::SD - 1) mbar_arrive(&sm.wu_empty[(q - (wu::SD - 1)) % wu::NS]);
      }
    }
    asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
    // the last SD - 1 chunks' slots (their stores have now completed)
    for (int j = (q > wu::SD - 1 ? q - (wu::SD - 1) : 0); j < q; ++j) mbar_arrive(&sm.wu_empty[j % wu::NS]);
  } else if (warp >= 4) {
    // ---------------- epilogue ----------------
    // The epilogue warps do not wait for one another: each waits for the accumulator and for
    // each chunk itself and hands the chunk on (and, after a tile's last chunk, the accumulator
    // back) with one mbarrier arrival per warp, so warps at different points of the chunk
    // sequence overlap their latencies.  No warp can get a ring's length ahead: a slot comes
    // back only after all of them have arrived.
    const int quarter = warp & 3;
    const int part = (warp - 4) >> 2;   // which CPT columns of each chunk
    const int r = quarter * 32 + lane;  // tile row of this thread
    const SgdParams& sp = args.sgd;
    // Every lane polls (acquiring what the barrier guards); the warp goes on only if all lanes
    // saw the phase, so a wait that runs out never splits the warp-wide tensor-memory
    // instructions that follow.
    auto warp_wait = [&](uint64_t* bar, uint32_t parity) -> bool {
      const bool okl = mbar_wait(bar, parity);
      return __all_sync(0xffffffffu, okl);
    };
    const float Gf = (float)args.G;
    const bool pow2 = (args.G & (args.G - 1)) == 0;
    const float invG = 1.0f / Gf;  // exact when G is a power of two
    // the update rule (0: no momentum, 1: heavy ball, 2: Nesterov); momentum implies u
    const int rule = sp.mom == 0.f ? 0 : (sp.nesterov ? 2 : 1);
    // This thread's CPT columns of a chunk, through the variant of wu_part_chunk for this launch's
    // rule and sign option and this tile's place in its unit: one branch per chunk, none per
    // element.
    auto part_chunk = [&](const float (&gv)[wu::CPT], float (&sc)[2 * wu::CPT], uint8_t* wrow,
                          uint8_t* urow, uint8_t* brow, bool first, bool last) {
      auto by_mode = [&](auto sg_tag, auto rule_tag) {
        constexpr bool SG = decltype(sg_tag)::value;
        constexpr int R = decltype(rule_tag)::value;
        if (!avg)
          wu_part_chunk<SG, R, wu::kPlain>(gv, sc, wrow, urow, brow, part, r, sp, Gf, invG, pow2);
        else if (first && last)
          wu_part_chunk<SG, R, wu::kAvg | wu::kFirst | wu::kLast>(gv, sc, wrow, urow, brow, part, r,
                                                                  sp, Gf, invG, pow2);
        else if (first)
          wu_part_chunk<SG, R, wu::kAvg | wu::kFirst>(gv, sc, wrow, urow, brow, part, r, sp, Gf,
                                                      invG, pow2);
        else if (last)
          wu_part_chunk<SG, R, wu::kAvg | wu::kLast>(gv, sc, wrow, urow, brow, part, r, sp, Gf,
                                                     invG, pow2);
        else
          wu_part_chunk<SG, R, wu::kAvg>(gv, sc, wrow, urow, brow, part, r, sp, Gf, invG, pow2);
      };
      auto by_rule = [&](auto sg_tag) {
        if (rule == 0)
          by_mode(sg_tag, std::integral_constant<int, 0>{});
        else if (rule == 1)
          by_mode(sg_tag, std::integral_constant<int, 1>{});
        else
          by_mode(sg_tag, std::integral_constant<int, 2>{});
      };
      if (sp.sign)
        by_rule(std::true_type{});
      else
        by_rule(std::false_type{});
    };
    int q = 0, i = 0;
    bool ok = true;
    for (; i < my_count && ok; ++i) {
      const WgradUpdateLayer* ly;
      int g, m0, n0, gi;
      tile_at(i, ly, g, m0, n0, gi);
      const bool first = gi == 0, last = gi == per_unit - 1;
      const int ab = i & 1;
      const int nc = wu_chunks(ly->N, n0);
      if (!warp_wait(&sm.acc_full[ab], (i >> 1) & 1)) {
        ok = false;
        break;
      }
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      for (int c = 0; c < nc; ++c, ++q) {
        const int sl = q % wu::NS;
        if (!warp_wait(&sm.wu_full[sl], (q / wu::NS) & 1)) {
          ok = false;
          break;
        }
        const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
        const uint32_t g_col = (uint32_t)(ab * wu::TN + c * wu::CW + wu::CPT * part);
        // averaging mode: this thread's running pair of the chunk over the replicas so far,
        // 2 CPT columns from 256 + 64 chunk + 2 CPT part (s in sc[0 .. CPT), c after it)
        const uint32_t sc_col = 2u * wu::TN + (uint32_t)(c * 2 * wu::CW + 2 * wu::CPT * part);
        float gv[wu::CPT], sc[2 * wu::CPT];
        if (avg && !first) {
          tmem_wait_st();  // this chunk's pair, stored at the previous replica
          tmem_ld_g8_sc16(tmem + lane_base + g_col, tmem + lane_base + sc_col, gv, sc);
        } else {
          tmem_ld8(tmem + lane_base + g_col, gv);
        }
        uint8_t* wrow = sm.w[sl] + r * 128;
        uint8_t* urow = sm.u[sl] + r * 128;
        uint8_t* brow = sm.wb[sl] + r * 64;
        part_chunk(gv, sc, wrow, urow, brow, first, last);
        if (avg && !last) tmem_st16_nowait(tmem + lane_base + sc_col, sc);
        // this warp's shared-memory writes reach the TMA stores, its accumulator reads are done
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(&sm.st_full[sl]);  // the store issuer takes the chunk once all warps have
          if (c == nc - 1) mbar_arrive(&sm.acc_empty[ab]);  // ... and the MMA the accumulator
        }
      }
    }
    tmem_wait_st();  // no tensor-memory store outstanding when the columns are freed
    (void)ok;
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (warp == 2) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(tmem_cols)
                 : "memory");
  }
}

// =============================================================================================
// Implicit-GEMM 3x3 convolution, persistent: out[g][p][n] = sum over taps t and k < ck of
// in[g][shift_t(p)][k] w[g][n][t][k] (zero padding 1, stride 1 or 2), fp32 out.
//
// A CTA owns one replica and every cpr-th 128-pixel tile of it.  The replica's weights (all nine
// taps, N rows of ck channels) are loaded once; the input streams through a ring of shared-memory
// stages by TMA (rank-5 boxes of the NHWC input, out-of-bounds fill = the zero padding, element
// strides = the convolution stride); two TMEM accumulators let a tile's MMAs overlap the previous
// tile's epilogue.  Two stage forms:
//   strip (stride 1, a tile = whole rows of one image): one stage per tile holds, for each kw, the
//     tile's rows plus one halo row above and below, shifted by kw - 1 columns; tap (kh, kw) is
//     that box from row kh on (a whole number of swizzle atoms further), so 3 boxes serve 9 taps;
//   per kernel row: three stages per tile, stage kh holds the three kw-shifted boxes of the
//     tile's rows under kernel row kh (stride 2, and tiles that span several images).
//   warp 0      TMA producer (weights once, then one stage per tap)
//   warp 1      MMA issuer: per tap ck / 16 tcgen05.mma (M = 128, N = NP, K = 16), descriptors
//               from precomputed bases (the issuing thread is on the critical path); with
//               nsplit = 3 the taps of column kw accumulate into partial kw, consecutive MMAs
//               into different partials (small-N MMAs into one accumulator wait on each other)
//   warp 2      TMEM allocation
//   warps 4-7   epilogue: tcgen05.ld of the tile row's NP columns (the partials' sum), fp32
//               stores
// nacc accumulator buffers (each nsplit x NP columns) let the MMAs of the next tiles run while
// the epilogue drains this one.
namespace cv {
constexpr int THREADS = 256;
constexpr int RING_BYTES = 96 * 1024;
constexpr int MAX_STAGES = 24;  // 4 KB stages (ck = 16)
constexpr int EPI0 = 128;
constexpr size_t SMEM_MAX = 227 * 1024;  // dynamic shared memory of one CTA
constexpr int MAX_ACC = 4;  // accumulator buffers in TMEM
// barriers, TMEM slot (16 bytes), and the BatchNorm-backward epilogue's mean / rstd (64 each)
constexpr size_t AUX_BYTES = (2 * MAX_STAGES + 2 * MAX_ACC + 1) * 8 + 16 + 2 * 64 * 4;
}  // namespace cv


__global__ void __launch_bounds__(cv::THREADS, 2) conv_tc_kernel(const __grid_constant__ ConvArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  const int ck = a.ck, np = a.np;
  // per-kernel-row form: a stage holds the three taps of one kernel row (three TMA boxes, one
  // handshake); strip form: a stage holds the three kw boxes of (rows + 2) image rows
  const uint32_t tap_bytes = (uint32_t)BM * ck * 2;
  const uint32_t row_bytes = (uint32_t)a.wout * ck * 2;  // one image row of the input box
  const uint32_t box_bytes = a.strip ? tap_bytes + 2 * row_bytes : tap_bytes;
  const uint32_t stage_bytes = 3 * box_bytes;
  const int spt = a.strip ? 1 : 3;  // stages per tile
  const int nst = min(cv::MAX_STAGES, a.ring_bytes / (int)stage_bytes);
  uint8_t* ring = base;
  uint8_t* wsm = base + a.ring_bytes;
  const uint32_t wtap = (uint32_t)np * ck * 2;  // bytes of one tap's weights
  uint64_t* bars = reinterpret_cast<uint64_t*>(wsm + 9 * wtap);
  uint64_t* full = bars;
  uint64_t* empty = bars + cv::MAX_STAGES;
  uint64_t* acc_full = bars + 2 * cv::MAX_STAGES;
  uint64_t* acc_empty = acc_full + cv::MAX_ACC;
  uint64_t* w_full = acc_empty + cv::MAX_ACC;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(w_full + 1);
  float* bw_mu = reinterpret_cast<float*>(tmem_slot + 4);  // [64]
  float* bw_rs = bw_mu + 64;                                // [64]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = blockIdx.y, cpr = gridDim.x;
  const int tiles = a.P / BM;  // per replica
  const int per_img = a.hout * a.wout;
  const int nacc = a.nacc, nsplit = a.nsplit;
  const uint32_t acc_cols = (uint32_t)(nsplit * np);  // one accumulator buffer
  const uint32_t tmem_cols = conv_tmem_cols(nacc * nsplit, np);

  if (threadIdx.x == 0) {
    for (int i = 0; i < nst; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < nacc; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], 4);  // one arrival per epilogue warp
    }
    mbar_init(w_full, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 2) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_slot)),
                 "r"(tmem_cols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;
  pdl_begin();  // everything above touched only shared memory and TMEM

  if (warp == 0 && lane == 0) {
    // ---------------- producer ----------------
    mbar_expect_tx(w_full, 9 * wtap);
    for (int t = 0; t < 9; ++t) tma_load_3d(wsm + t * wtap, &a.w_map, w_full, t * ck, 0, g);
    int q = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < tiles && ok; tile += cpr) {
      const int p0 = tile * BM, b0 = p0 / per_img, oy0 = (p0 / a.wout) % a.hout;
      for (int sp = 0; sp < spt; ++sp, ++q) {
        const int sl = q % nst;
        if (!mbar_wait(&empty[sl], ((q / nst) & 1) ^ 1)) {
          ok = false;
          break;
        }
        mbar_expect_tx(&full[sl], stage_bytes);
        // strip: rows oy0 - 1 .. oy0 + rows (the halo rows out of the image read as zeros);
        // per kernel row sp: the rows under kernel row sp
        const int y0 = a.strip ? oy0 - 1 : oy0 * a.stride + sp - 1;
        for (int kw = 0; kw < 3; ++kw)
          tma_load_5d(ring + sl * stage_bytes + kw * box_bytes, &a.in_map, &full[sl], 0, kw - 1,
                      y0, b0, g);
      }
    }
    // copies in flight land before the CTA can exit
    mbar_wait(w_full, 0);
    for (int j = (q > nst ? q - nst : 0); j < q; ++j) mbar_wait(&full[j % nst], (j / nst) & 1);
  } else if (warp == 1 && lane == 0) {
    // ---------------- MMA issuer ----------------
    const uint32_t idesc = make_idesc(BM, np, false, false);
    const uint32_t swz = (uint32_t)ck * 2;
    // descriptors of the ring's start and of tap 0's weights: the address field is in 16-byte
    // units, so the descriptor of a tap / stage / K-step is the base plus its byte offset / 16
    const uint64_t a_desc0 = smem_desc_kmajor(smem_u32(ring), swz);
    const uint64_t b_desc0 = smem_desc_kmajor(smem_u32(wsm), swz);
    const uint32_t kw_step = box_bytes >> 4, kh_step = (a.strip ? row_bytes : 0u) >> 4;
    const uint32_t tap_step = wtap >> 4;
    bool ok = mbar_wait(w_full, 0);
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    int q = 0, i = 0;
    for (int tile = blockIdx.x; tile < tiles && ok; tile += cpr, ++i) {
      const int ab = i % nacc;
      if (!mbar_wait(&acc_empty[ab], ((i / nacc) & 1) ^ 1)) break;
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const uint32_t acc = tmem + (uint32_t)ab * acc_cols;
      for (int sp = 0; sp < spt; ++sp, ++q) {
        const int sl = q % nst;
        if (!mbar_wait(&full[sl], (q / nst) & 1)) {
          ok = false;
          break;
        }
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint64_t st_desc = a_desc0 + ((uint32_t)sl * stage_bytes >> 4);
        for (int kh = a.strip ? 0 : sp; kh < (a.strip ? 3 : sp + 1); ++kh) {
          const uint64_t row_desc = st_desc + (uint32_t)kh * kh_step;
          for (int kk = 0; kk < ck / 16; ++kk) {
#pragma unroll
            for (int kw = 0; kw < 3; ++kw) {
              const int t = kh * 3 + kw;
              // partial kw (nsplit = 3) starts at its first kernel row; a single accumulator at
              // the first tap
              const bool first = kk == 0 && (nsplit == 3 ? kh == 0 : t == 0);
              mma_bf16(acc + (nsplit == 3 ? (uint32_t)(kw * np) : 0u),
                       row_desc + (uint32_t)kw * kw_step + (uint32_t)(2 * kk),
                       b_desc0 + (uint32_t)t * tap_step + (uint32_t)(2 * kk), idesc,
                       first ? 0u : 1u);
            }
          }
        }
        // strip form: the epilogue releases the stage once it sees the tile's accumulator (one
        // commit per tile); per kernel row: the stage is released as soon as its MMAs complete
        if (!a.strip) mma_commit(&empty[sl]);
      }
      if (ok) mma_commit(&acc_full[ab]);
    }
  } else if (warp >= 4) {
    // ---------------- epilogue ----------------
    // The four epilogue warps do not wait for one another: each waits for a tile's accumulator
    // itself (every lane polls; the warp goes on only if all lanes saw the phase, so a wait that
    // runs out never splits a warp-wide tensor-memory load) and gives it back with one arrival.
    const int quarter = warp & 3, r = quarter * 32 + lane;
    auto warp_wait = [&](uint64_t* bar, uint32_t parity) -> bool {
      const bool okl = mbar_wait(bar, parity);
      return __all_sync(0xffffffffu, okl);
    };
    // per-channel BatchNorm statistics of the output pixels (forward convolutions), per
    // epilogue warp: lanes 2 j, 2 j + 1 keep channel 16 ci + j's running count, mean and M2 over
    // the warp's 32 rows of every tile
    const bool with_stats = a.stats != nullptr;
    float run_n = 0.f, run_mu[4] = {0.f, 0.f, 0.f, 0.f}, run_m2[4] = {0.f, 0.f, 0.f, 0.f};
    // the data gradient's BatchNorm-backward epilogue (a.bwd): that layer's mean and rstd in
    // shared memory; lanes 2 j, 2 j + 1 keep channel 16 ci + j's running sums of g and g xhat
    const ConvBwdFuse& bw = a.bwd;
    const bool with_bwd = bw.y != nullptr;
    const int dx_h = a.dst_h > 0 ? a.dst_h : a.hout, dx_w = a.dst_w > 0 ? a.dst_w : a.wout;
    float run_g[4] = {0.f, 0.f, 0.f, 0.f}, run_gx[4] = {0.f, 0.f, 0.f, 0.f};
    if (with_bwd) {
      const int et = threadIdx.x - cv::EPI0;
      if (et < a.N) {
        bw_mu[et] = bw.mean[g * a.N + et];
        bw_rs[et] = bw.rstd[g * a.N + et];
      }
      asm volatile("bar.sync 1, 128;" ::: "memory");
    }
    int i = 0;
    for (int tile = blockIdx.x; tile < tiles; tile += cpr, ++i) {
      const int ab = i % nacc;
      if (!warp_wait(&acc_full[ab], (i / nacc) & 1)) break;
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      // strip form: this tile's MMAs (and so its reads of its input stage) are complete
      if (a.strip && quarter == 0 && lane == 0) mbar_arrive(&empty[i % nst]);
      int64_t dst = (int64_t)tile * BM + r;
      if (a.dst_h > 0) {
        const int pp = tile * BM + r, img = pp / per_img, rem = pp - img * per_img;
        const int oy = rem / a.wout, ox = rem - oy * a.wout;
        dst = ((int64_t)img * a.dst_h + 2 * oy + a.ph_y) * a.dst_w + 2 * ox + a.ph_x;
      }
      float* orow = a.out + (int64_t)g * a.out_gs + dst * a.N;
      // the shortcut's source pixel in the block output (stride 1: the same pixel; stride 2: the
      // pixels on the stride grid), or -1
      auto sc_pixel = [&](int64_t d) -> int64_t {
        if (!bw.sc_dout) return -1;
        const int img = (int)(d / ((int64_t)dx_h * dx_w)), rem = (int)(d % ((int64_t)dx_h * dx_w));
        const int iy = rem / dx_w, ix = rem - iy * dx_w;
        if (bw.sc_stride == 1) return d;
        if ((iy & 1) || (ix & 1)) return -1;
        return ((int64_t)img * (dx_h / 2) + iy / 2) * (dx_w / 2) + ix / 2;
      };
      int64_t sc_px = with_bwd ? sc_pixel(dst) : -1;
      if (with_bwd && tile + cpr < tiles) {
        // this thread's row of the next tile into L1 while this tile is processed: the loads
        // below would otherwise each wait on DRAM
        const int nt = tile + cpr;
        int64_t nd = (int64_t)nt * BM + r;
        if (a.dst_h > 0) {
          const int pp = nt * BM + r, img = pp / per_img, rem = pp - img * per_img;
          const int oy = rem / a.wout, ox = rem - oy * a.wout;
          nd = ((int64_t)img * a.dst_h + 2 * oy + a.ph_y) * a.dst_w + 2 * ox + a.ph_x;
        }
        const int64_t ne = (int64_t)g * a.out_gs + nd * a.N;
        for (int b = 0; b < a.N * 2; b += 128)
          asm volatile("prefetch.global.L1 [%0];" ::"l"(reinterpret_cast<const char*>(bw.mask + ne) + b));
        for (int b = 0; b < a.N * 4; b += 128)
          asm volatile("prefetch.global.L1 [%0];" ::"l"(reinterpret_cast<const char*>(bw.y + ne) + b));
        const int64_t ns = sc_pixel(nd);
        if (ns >= 0) {
          const int64_t se = (int64_t)g * bw.sc_gs + ns * bw.sc_C;
          for (int b = 0; b < a.N * 4; b += 128)
            asm volatile("prefetch.global.L1 [%0];" ::"l"(reinterpret_cast<const char*>(bw.sc_dout + se) + b));
          for (int b = 0; b < a.N * 2; b += 128)
            asm volatile("prefetch.global.L1 [%0];" ::"l"(reinterpret_cast<const char*>(bw.sc_out + se) + b));
        }
      }
#pragma unroll
      for (int ci = 0; ci < 4; ++ci) {
        const int c0 = 16 * ci;
        if (c0 >= a.N) break;
        float v[16];
        const uint32_t tl = tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)ab * acc_cols + c0;
        tmem_ld16(tl, v);
        if (nsplit == 3) {
          // the three column partials, added in column order
#pragma unroll
          for (int kw = 1; kw < 3; ++kw) {
            float u[16];
            tmem_ld16(tl + (uint32_t)(kw * np), u);
#pragma unroll
            for (int j = 0; j < 16; ++j) v[j] += u[j];
          }
        }
        if (with_bwd) {
          // dx (+ the shortcut's share) masked by the layer below's ReLU, and that layer's
          // BatchNorm-backward sums over this warp's rows
          if (sc_px >= 0) {
            const float4* sd = reinterpret_cast<const float4*>(
                bw.sc_dout + (int64_t)g * bw.sc_gs + sc_px * bw.sc_C + c0);
            const uint4* so = reinterpret_cast<const uint4*>(
                bw.sc_out + (int64_t)g * bw.sc_gs + sc_px * bw.sc_C + c0);
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const uint4 o8 = __ldg(so + h);
              const float4 d0 = __ldg(sd + 2 * h), d1 = __ldg(sd + 2 * h + 1);
              const uint32_t ow[4] = {o8.x, o8.y, o8.z, o8.w};
              const float dd[8] = {d0.x, d0.y, d0.z, d0.w, d1.x, d1.y, d1.z, d1.w};
#pragma unroll
              for (int k = 0; k < 8; ++k) {
                const float o = bf2f((uint16_t)(k & 1 ? ow[k >> 1] >> 16 : ow[k >> 1] & 0xffffu));
                v[8 * h + k] += o > 0.f ? dd[k] : 0.f;
              }
            }
          }
          const uint4* mk = reinterpret_cast<const uint4*>(bw.mask + (int64_t)g * a.out_gs + dst * a.N + c0);
          const float4* yv = reinterpret_cast<const float4*>(bw.y + (int64_t)g * a.out_gs + dst * a.N + c0);
          float gx[16];
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const uint4 m8 = __ldg(mk + h);
            const float4 y0 = __ldg(yv + 2 * h), y1 = __ldg(yv + 2 * h + 1);
            const uint32_t mw[4] = {m8.x, m8.y, m8.z, m8.w};
            const float yy[8] = {y0.x, y0.y, y0.z, y0.w, y1.x, y1.y, y1.z, y1.w};
#pragma unroll
            for (int k = 0; k < 8; ++k) {
              const int j = 8 * h + k;
              const float m = bf2f((uint16_t)(k & 1 ? mw[k >> 1] >> 16 : mw[k >> 1] & 0xffffu));
              v[j] = m > 0.f ? v[j] : 0.f;
              gx[j] = v[j] * ((yy[k] - bw_mu[c0 + j]) * bw_rs[c0 + j]);
            }
          }
          float t[16];
#pragma unroll
          for (int j = 0; j < 16; ++j) t[j] = v[j];
          run_g[ci] += warp_colsum16(t, lane);
          run_gx[ci] += warp_colsum16(gx, lane);
        }
        if (a.st32) {
          // whole 32-byte sectors per lane and instruction
#pragma unroll
          for (int j = 0; j < 2; ++j)
            asm volatile("st.global.v8.f32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(
                             orow + c0 + 8 * j),
                         "f"(v[8 * j]), "f"(v[8 * j + 1]), "f"(v[8 * j + 2]), "f"(v[8 * j + 3]),
                         "f"(v[8 * j + 4]), "f"(v[8 * j + 5]), "f"(v[8 * j + 6]), "f"(v[8 * j + 7])
                         : "memory");
        } else {
#pragma unroll
          for (int j = 0; j < 4; ++j)
            *reinterpret_cast<float4*>(orow + c0 + 4 * j) =
                make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
        }
        if (with_stats) {
          // this warp's 32 pixels of the tile: mean, then the sum of squared deviations from
          // it (two passes over the registers), each summed over the warp's lanes
          float t[16];
#pragma unroll
          for (int j = 0; j < 16; ++j) t[j] = v[j];
          const float mt = warp_colsum16(t, lane) * (1.f / 32);
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const float e = v[j] - __shfl_sync(0xffffffffu, mt, 2 * j);
            t[j] = e * e;
          }
          const float m2t = warp_colsum16(t, lane);
          // Chan et al.'s combination of the running (n, mean, M2) with these 32 pixels'
          const float nt = run_n + 32.f, f = 32.f / nt, delta = mt - run_mu[ci];
          run_mu[ci] = fmaf(delta, f, run_mu[ci]);
          run_m2[ci] = run_m2[ci] + m2t + delta * delta * run_n * f;
        }
      }
      if (with_stats) run_n += 32.f;
      asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[ab]);
    }
    if (with_bwd && !(lane & 1)) {
#pragma unroll
      for (int ci = 0; ci < 4; ++ci) {
        if (16 * ci >= a.N) break;
        bw.part[((int64_t)g * bw.part_gs + bw.part_off + 4 * blockIdx.x + quarter) * a.N + 16 * ci +
                (lane >> 1)] = make_float2(run_g[ci], run_gx[ci]);
      }
    }
    if (with_stats && !(lane & 1)) {
      // one partial per epilogue warp: stats[g][4 q + quarter]
#pragma unroll
      for (int ci = 0; ci < 4; ++ci) {
        if (16 * ci >= a.N) break;
        a.stats[((int64_t)g * cpr * 4 + 4 * blockIdx.x + quarter) * a.N + 16 * ci + (lane >> 1)] =
            make_float4(run_n, run_mu[ci], run_m2[ci], 0.f);
      }
    }
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (warp == 2) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(tmem_cols)
                 : "memory");
  }
}


// =============================================================================================
// Weight gradient of a 3x3 convolution on the tensor cores, column matrix built in shared memory:
//   dW[g][co][t][ci] = sum over output pixels p of dy[g][p][co] x[g][src_t(p)][ci].
// As D[m][n] = sum_k A[m][k] B[n][k] with m = t Cin + ci (9 Cin rows in 128-row tiles), n = co
// (one 64-wide operand, zero beyond Cout) and k = output pixels in blocks of 64: B is the output
// gradient's 64 x 64 tile by TMA (pixel-major = MN-major, 128-byte swizzle); A is MN-major too,
// gathered by the builder warps from a TMA-loaded strip of input rows (the halo rows above and
// below come from out-of-bounds zero fill, the halo columns are written as zeros): one 16-byte
// chunk = 8 channels of one tap and pixel per copy.  A CTA owns one replica and a contiguous range
// of pixel blocks and keeps every m-tile's 128 x 64 fp32 accumulator in TMEM; it writes its
// partial dW, and a second kernel sums the CTAs' partials in order.  Rows m >= 9 Cin of the last
// m-tile are never written: they only reach accumulator rows that are not stored.
// Two rings: the small TMA inputs (strip + tile) run `ni` blocks ahead, and `na` A tiles
// (two to four) let the builders run ahead of the MMAs.
//   warp 0      TMA producer (input strip + output-gradient tile per block)
//   warp 1      MMA issuer: per block and m-tile, 4 x tcgen05.mma (M = 128, N = 64, K = 16)
//   warp 2      TMEM allocation
//   warps 4-7   build A for each block; at the end, tcgen05.ld of the accumulators and the
//               partial's stores
namespace cw {
constexpr int THREADS = 384;
constexpr int MAX_NA = 4;   // A buffers
constexpr int MAX_NI = 16;  // input stages
constexpr int KB = 64;      // output pixels per block
constexpr int BUILDERS = 8; // builder warps (warps 4-11)
constexpr int MAX_CH = 18;  // 16-byte chunks per builder thread (9 taps x Cin / 8 / 4 parts)
constexpr int MAX_MT = 5;   // m-tiles (9 Cin <= 640)
constexpr uint32_t kTileA = 16384;  // one m-tile of A: two 64-row atoms x 64 pixels x 128 B
constexpr uint32_t kTileB = 8192;   // the output-gradient tile: 64 pixels x 128 B
constexpr uint32_t kTwoPerSm = 113 * 1024;  // shared memory that still fits two CTAs on an SM
constexpr uint32_t kOnePerSm = 224 * 1024;
}  // namespace cw

__host__ __device__ inline int cw_rows(int stride, int wout) { return (cw::KB / wout - 1) * stride + 3; }
__host__ __device__ inline uint32_t cw_halo_pitch(int cin, int stride, int win, int wout) {
  return ((uint32_t)cw_rows(stride, wout) * win * cin * 2 + 1023u) & ~1023u;
}

__global__ void __launch_bounds__(cw::THREADS, 1) conv_wgrad_tc_kernel(
    const __grid_constant__ ConvWgradArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  const int cin = a.cin, cout = a.cout, mrows = 9 * cin, ni = a.ni, na = a.na;
  const int mt_n = (mrows + 127) / 128;
  const int rh = cw_rows(a.stride, a.wout);
  const uint32_t halo_bytes = (uint32_t)rh * a.win * cin * 2;
  const uint32_t in_pitch = cw_halo_pitch(cin, a.stride, a.win, a.wout) + cw::kTileB;
  const uint32_t a_bytes = (uint32_t)mt_n * cw::kTileA;
  uint8_t* A0 = base;                          // [na][mt_n][2][64][128 B]
  uint8_t* I0 = A0 + na * a_bytes;             // [ni]: output-gradient tile, then the strip
  uint64_t* full_in = reinterpret_cast<uint64_t*>(I0 + ni * in_pitch);
  uint64_t* empty_in = full_in + cw::MAX_NI;   // arrivals: the MMAs (tile), each builder (strip)
  uint64_t* aready = empty_in + cw::MAX_NI;
  uint64_t* afree = aready + cw::MAX_NA;
  uint64_t* acc_full = afree + cw::MAX_NA;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_full + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = blockIdx.y, q = blockIdx.x, cpr = gridDim.x;
  const int nkb = a.P / cw::KB;
  const int kb0 = (int)((int64_t)q * nkb / cpr);
  const int nblk = (int)((int64_t)(q + 1) * nkb / cpr) - kb0;
  const int per_img = a.hout * a.wout;
  const int nb = a.nb;                               // MMA N: output-gradient channels
  const uint32_t tile_b = (uint32_t)cw::KB * nb * 2;  // bytes of the output-gradient tile
  uint32_t tmem_cols = 32;
  while (tmem_cols < (uint32_t)(mt_n * nb)) tmem_cols <<= 1;

  if (threadIdx.x == 0) {
    for (int i = 0; i < ni; ++i) {
      mbar_init(&full_in[i], 1);
      mbar_init(&empty_in[i], 1 + cw::BUILDERS);
    }
    for (int i = 0; i < na; ++i) {
      mbar_init(&aready[i], cw::BUILDERS);
      mbar_init(&afree[i], 1);
    }
    mbar_init(acc_full, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 2) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_slot)),
                 "r"(tmem_cols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;
  pdl_begin();  // everything above touched only shared memory and TMEM

  if (warp == 0 && lane == 0) {
    // ---------------- producer ----------------
    int j = 0;
    for (; j < nblk; ++j) {
      const int s = j % ni;
      if (!mbar_wait(&empty_in[s], ((j / ni) & 1) ^ 1)) break;
      const int p0 = (kb0 + j) * cw::KB;
      const int b = p0 / per_img, oy0 = (p0 % per_img) / a.wout;
      uint8_t* st = I0 + s * in_pitch;
      mbar_expect_tx(&full_in[s], halo_bytes + tile_b);
      tma_load_3d(st, &a.dy_map, &full_in[s], 0, p0, g);
      tma_load_5d(st + cw::kTileB, &a.x_map, &full_in[s], 0, 0, oy0 * a.stride - 1, b, g);
    }
    // copies in flight land before the CTA can exit
    for (int i = (j > ni ? j - ni : 0); i < j; ++i) mbar_wait(&full_in[i % ni], (i / ni) & 1);
  } else if (warp == 1 && lane == 0) {
    // ---------------- MMA issuer ----------------
    const uint32_t idesc = make_idesc(BM, nb, true, true);
    // descriptors of A0 and I0; a buffer / m-tile / K-step adds its byte offset / 16.  B: rows of
    // 2 nb bytes (nb channels) swizzled at that width, 8-row groups 16 nb bytes apart, K-steps of
    // 16 pixels 32 nb bytes apart; one swizzle atom spans all nb channels.
    const uint64_t a_desc0 = smem_desc(smem_u32(A0), 8192, 1024);
    const uint64_t b_desc0 = nb == 64 ? smem_desc(smem_u32(I0), 8192, 1024)
                                      : smem_desc_swz(smem_u32(I0), 16u * nb, 16u * nb, 2u * nb);
    bool ok = true;
    for (int j = 0; j < nblk; ++j) {
      const int s = j % ni, sa = j % na;
      if (!mbar_wait(&aready[sa], (j / na) & 1) || !mbar_wait(&full_in[s], (j / ni) & 1)) {
        ok = false;
        break;
      }
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const uint64_t ad = a_desc0 + ((uint32_t)sa * a_bytes >> 4);
      const uint64_t bd = b_desc0 + ((uint32_t)s * in_pitch >> 4);
      for (int mt = 0; mt < mt_n; ++mt)
#pragma unroll
        for (int kk = 0; kk < cw::KB / 16; ++kk)
          mma_bf16(tmem + (uint32_t)(mt * nb), ad + (uint32_t)(mt * (cw::kTileA >> 4) + kk * 128),
                   bd + (uint32_t)(kk * 2 * nb), idesc, (j > 0 || kk > 0) ? 1u : 0u);
      mma_commit(&afree[sa]);    // A buffer reusable once these MMAs have read it
      mma_commit(&empty_in[s]);  // and the output-gradient tile
    }
    if (ok && nblk > 0) mma_commit(acc_full);
  } else if (warp >= 4) {
    // ---------------- builders, then the epilogue ----------------
    // Builder thread = (pixel k of the block, part p of 4): it copies chunks p, p + 4, ... of the
    // pixel's 9 Cin / 8 sixteen-byte chunks (tap t, channels 8 cg..8 cg + 7).  Where each of them
    // comes from in the strip and goes to in A is the same for every block, so the offsets are
    // worked out once; per block a thread does at most MAX_CH loads and stores.  Each warp waits
    // and signals by itself (aready and empty_in count the warps), with two warps per scheduler
    // so that one's load latency hides behind the other's work.
    const int bt = threadIdx.x - 128;
    const int k = bt & (cw::KB - 1), part = bt >> 6;
    const int cg_n = cin / 8, nchunk = 9 * cg_n;
    const int r = k / a.wout, ox = k - r * a.wout;
    const uint32_t swz_mask = cin == 64 ? 7u : (cin == 32 ? 3u : 1u);  // the strip's swizzle
    uint32_t src_off[cw::MAX_CH], dst_off[cw::MAX_CH];
    uint32_t inside = 0;
    int nch = 0;
#pragma unroll
    for (int i = 0; i < cw::MAX_CH; ++i) {
      const int c = part + 4 * i;
      src_off[i] = dst_off[i] = 0;
      if (c < nchunk) {
        const int t = c / cg_n, cg = c - t * cg_n;
        const int kh = t / 3, kw = t - 3 * kh;
        const int ix = ox * a.stride + kw - 1;
        if (ix >= 0 && ix < a.win) {
          const uint32_t o = (uint32_t)(((r * a.stride + kh) * a.win + ix) * cin) * 2u + (uint32_t)cg * 16u;
          src_off[i] = o ^ (((o >> 7) & swz_mask) << 4);
          inside |= 1u << i;
        }
        const int m = t * cin + cg * 8;
        dst_off[i] = (uint32_t)(m >> 7) * cw::kTileA + (uint32_t)((m >> 6) & 1) * 8192u +
                     (uint32_t)(k >> 3) * 1024u + (uint32_t)(k & 7) * 128u +
                     ((uint32_t)(((m >> 3) & 7) ^ (k & 7)) << 4);
        nch = i + 1;
      }
    }
    auto wwait = [&](uint64_t* bar, uint32_t parity) -> bool {
      return __all_sync(0xffffffffu, mbar_wait(bar, parity) ? 1 : 0) != 0;
    };
    bool ok = true;
    for (int j = 0; j < nblk; ++j) {
      const int s = j % ni, sa = j % na;
      if (!wwait(&full_in[s], (j / ni) & 1) || !wwait(&afree[sa], ((j / na) & 1) ^ 1)) {
        ok = false;
        break;
      }
      const uint32_t X = smem_u32(I0 + s * in_pitch + cw::kTileB);
      const uint32_t A = smem_u32(A0 + sa * a_bytes);
#pragma unroll
      for (int i = 0; i < cw::MAX_CH; ++i) {
        if (i < nch) {
          uint32_t v0 = 0u, v1 = 0u, v2 = 0u, v3 = 0u;
          if (inside & (1u << i))
            asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                         : "=r"(v0), "=r"(v1), "=r"(v2), "=r"(v3)
                         : "r"(X + src_off[i])
                         : "memory");
          asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(A + dst_off[i]), "r"(v0),
                       "r"(v1), "r"(v2), "r"(v3)
                       : "memory");
        }
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // visible to the MMAs
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&aready[sa]);
        mbar_arrive(&empty_in[s]);  // this warp has read the strip
      }
    }
    if (warp >= 8) ok = false;  // the epilogue: warps 4-7, one TMEM lane quarter each
    if (ok && nblk > 0 && wwait(acc_full, 0)) {
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const int quarter = warp & 3;
      float* out = a.part + ((int64_t)g * cpr + q) * cout * mrows;
      for (int mt = 0; mt < mt_n; ++mt) {
        const int m = mt * 128 + quarter * 32 + lane;
        for (int c0 = 0; c0 < cout; c0 += 16) {
          float v[16];
          tmem_ld16(tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(mt * nb + c0), v);
          if (m < mrows) {
#pragma unroll
            for (int i = 0; i < 16; ++i) out[(int64_t)(c0 + i) * mrows + m] = v[i];
          }
        }
      }
    }
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (warp == 2) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(tmem_cols)
                 : "memory");
  }
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;

void load_encode() {
  void* fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
          cudaSuccess &&
      q == cudaDriverEntryPointSuccess)
    g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  else
    cudaGetLastError();
}

template <int BN, int STAGES>
constexpr size_t smem_bytes() {
  return sizeof(Smem<BN, STAGES>) + 1024;
}

template <int BN, int STAGES>
cudaError_t launch_cfg(const TcGemmArgs& a, dim3 grid, cudaStream_t stream) {
  constexpr size_t smem = smem_bytes<BN, STAGES>();
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(gemm_tc_kernel<BN, STAGES>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  launch_pdl(gemm_tc_kernel<BN, STAGES>, grid, dim3(128), smem, stream, a);
  return cudaGetLastError();
}

}  // namespace

bool tc_available() {
  int dev = 0;
  cudaDeviceProp p;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaGetDeviceProperties(&p, dev) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  std::call_once(g_encode_once, load_encode);
  return p.major == 10 && g_encode != nullptr;
}

bool make_tma_map_f32(CUtensorMap* map, const void* base, uint64_t dim0, uint64_t dim1,
                      uint64_t dim2, uint64_t s1, uint64_t s2, uint32_t box0, uint32_t box1) {
  std::call_once(g_encode_once, load_encode);
  if (!g_encode) return false;
  if ((reinterpret_cast<uintptr_t>(base) & 15) || ((s1 * 4) & 15) || ((s2 * 4) & 15)) return false;
  cuuint64_t dims[3] = {dim0, dim1, dim2};
  cuuint64_t strides[2] = {s1 * 4, s2 * 4};
  cuuint32_t box[3] = {box0, box1, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, const_cast<void*>(base), dims,
                        strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

namespace {
// The expiry path of the GEMM's bounded waits, on its own: one thread waits on an mbarrier phase
// that completes only if `arrive` is set, through the same mbar_wait (limit in SM cycles).
// out = 1 if the phase completed, 0 if the wait ran out (g_tc_timeout is then set).
__global__ void bounded_wait_selftest_kernel(long long limit_cycles, int arrive, int* out) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x != 0) return;
  mbar_init(&bar, 1);
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  if (arrive) mbar_arrive(&bar);
  *out = mbar_wait(&bar, 0, limit_cycles) ? 1 : 0;
}
}  // namespace

cudaError_t launch_bounded_wait_selftest(long long limit_cycles, int arrive, int* out,
                                         cudaStream_t stream) {
  if (limit_cycles < 0 || limit_cycles > kWaitCycles || !out) return cudaErrorInvalidValue;
  bounded_wait_selftest_kernel<<<1, 32, 0, stream>>>(limit_cycles, arrive, out);
  return cudaGetLastError();
}

int tc_take_timeout_flag() {
  int h = 0;
  if (cudaMemcpyFromSymbol(&h, g_tc_timeout, sizeof(int)) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  if (h) {
    const int zero = 0;
    cudaMemcpyToSymbol(g_tc_timeout, &zero, sizeof(int));
  }
  return h;
}

bool make_tma_map_bf16(CUtensorMap* map, const void* base, uint64_t dim0, uint64_t dim1,
                       uint64_t dim2, uint64_t s1, uint64_t s2, uint32_t box0, uint32_t box1) {
  std::call_once(g_encode_once, load_encode);
  if (!g_encode) return false;
  if ((reinterpret_cast<uintptr_t>(base) & 15) || ((s1 * 2) & 15) || ((s2 * 2) & 15)) return false;
  cuuint64_t dims[3] = {dim0, dim1, dim2};
  cuuint64_t strides[2] = {s1 * 2, s2 * 2};
  cuuint32_t box[3] = {box0, box1, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims,
                        strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool make_tma_map(CUtensorMap* map, const void* base, bool bf16, uint64_t dim0, uint64_t dim1,
                  uint64_t dim2, uint64_t s1, uint64_t s2, uint32_t box0, uint32_t box1,
                  int swizzle_bytes) {
  std::call_once(g_encode_once, load_encode);
  if (!g_encode) return false;
  const uint64_t esz = bf16 ? 2 : 4;
  if ((reinterpret_cast<uintptr_t>(base) & 15) || ((s1 * esz) & 15) || ((s2 * esz) & 15)) return false;
  CUtensorMapSwizzle sw;
  switch (swizzle_bytes) {
    case 0: sw = CU_TENSOR_MAP_SWIZZLE_NONE; break;
    case 32: sw = CU_TENSOR_MAP_SWIZZLE_32B; break;
    case 64: sw = CU_TENSOR_MAP_SWIZZLE_64B; break;
    case 128: sw = CU_TENSOR_MAP_SWIZZLE_128B; break;
    default: return false;
  }
  if (swizzle_bytes && box0 * esz > (uint64_t)swizzle_bytes) return false;
  cuuint64_t dims[3] = {dim0, dim1, dim2};
  cuuint64_t strides[2] = {s1 * esz, s2 * esz};
  cuuint32_t box[3] = {box0, box1, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = g_encode(map, bf16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32,
                        3, const_cast<void*>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

namespace {
// The launch shape of conv_tc_kernel: false if the arguments are not taken.
bool conv_tc_plan(const ConvArgs& a, int sms, int* per_sm, size_t* ring, size_t* smem, int* cpr) {
  if (a.stats && a.dst_h > 0) return false;
  if (a.bwd.y && (!a.bwd.mask || !a.bwd.mean || !a.bwd.rstd || !a.bwd.part ||
                  (a.bwd.sc_dout && (!a.bwd.sc_out || a.bwd.sc_C < a.N ||
                                     (a.bwd.sc_stride != 1 && a.bwd.sc_stride != 2)))))
    return false;
  int rows = 0, images = 0;
  if ((a.ck != 16 && a.ck != 32 && a.ck != 64) || (a.stride != 1 && a.stride != 2) ||
      (a.N != 16 && a.N != 32 && a.N != 64) || a.np != a.N || !a.out || a.G > 65535 ||
      !conv_tile_shape(a.hout, a.wout, &rows, &images) || a.P % (a.hout * a.wout) || a.P % BM ||
      (a.dst_h > 0 && (a.dst_h < 2 * a.hout || a.dst_w < 2 * a.wout || a.ph_y < 0 || a.ph_y > 1 ||
                       a.ph_x < 0 || a.ph_x > 1)))
    return false;
  const size_t fixed = 1024 + 9 * (size_t)a.np * a.ck * 2 + cv::AUX_BYTES;
  const bool strip = a.strip != 0;
  if (strip && !conv_strip_ok(a.hout, a.wout, a.stride)) return false;
  const size_t stage_bytes = 3 * ((size_t)BM + (strip ? 2 * a.wout : 0)) * a.ck * 2;
  const size_t two_budget = 113 * 1024;
  *ring = cv::RING_BYTES;
  *per_sm = 1;
  if (two_budget > fixed && (two_budget - fixed) / stage_bytes >= 3) {
    *ring = std::min<size_t>(cv::RING_BYTES, ((two_budget - fixed) / 1024) * 1024);
    *per_sm = 2;
  }
  if (*per_sm == 1) {
    // one CTA per SM: the ring takes what the weights leave of the 227 KB (at most 24 stages)
    *ring = std::min<size_t>((size_t)cv::MAX_STAGES * stage_bytes,
                             ((cv::SMEM_MAX - fixed) / stage_bytes) * stage_bytes);
  }
  *smem = fixed + *ring;
  // CTAs per replica: as many as fit on the SMs at once over all replicas (one wave), at most one
  // per tile
  *cpr = std::max(1, std::min(a.P / BM, *per_sm * sms / a.G));
  return true;
}

int device_sms(int* sms) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(sms, cudaDevAttrMultiProcessorCount, dev);
  return e == cudaSuccess ? dev : -1;
}
}  // namespace

int conv_tc_ctas(const ConvArgs& a) {
  int sms = 0, per_sm = 1, cpr = 0;
  size_t ring = 0, smem = 0;
  if (a.P <= 0 || a.G <= 0 || device_sms(&sms) < 0) return 0;
  return conv_tc_plan(a, sms, &per_sm, &ring, &smem, &cpr) ? cpr : 0;
}

cudaError_t launch_conv_tc(const ConvArgs& a, cudaStream_t stream, int* ctas_per_replica) {
  if (a.P <= 0 || a.G <= 0) return cudaSuccess;
  int rows = 0, images = 0;
  if ((a.ck != 16 && a.ck != 32 && a.ck != 64) || (a.stride != 1 && a.stride != 2) ||
      (a.N != 16 && a.N != 32 && a.N != 64) || a.np != a.N || !a.out || a.G > 65535 ||
      !conv_tile_shape(a.hout, a.wout, &rows, &images) || a.P % (a.hout * a.wout) || a.P % BM ||
      (a.dst_h > 0 && (a.dst_h < 2 * a.hout || a.dst_w < 2 * a.wout || a.ph_y < 0 || a.ph_y > 1 ||
                       a.ph_x < 0 || a.ph_x > 1)))
    return cudaErrorInvalidValue;
  (void)rows;
  (void)images;
  // Two CTAs per SM where the weights leave room for a ring of at least three stages (a CTA's
  // tiles pass through a chain of handshakes one after another; two CTAs overlap their chains),
  // else one CTA with the full ring (conv_tc_plan).
  int sms = 0, per_sm = 1, cpr = 0;
  size_t ring = 0, smem = 0;
  const int dev = device_sms(&sms);
  if (dev < 0) return cudaErrorInvalidDevice;
  if (!conv_tc_plan(a, sms, &per_sm, &ring, &smem, &cpr)) return cudaErrorInvalidValue;
  cudaError_t e = cudaSuccess;
  ConvArgs la = a;
  la.ring_bytes = (int)ring;
  la.st32 = (reinterpret_cast<uintptr_t>(a.out) & 31) == 0 && a.out_gs % 8 == 0 ? 1 : 0;
  static int attr_dev = -1;
  if (attr_dev != dev) {
    e = cudaFuncSetAttribute(conv_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)cv::SMEM_MAX);
    if (e != cudaSuccess) return e;
    attr_dev = dev;
  }
  // accumulators (measured in the ResNet-20 step): four buffers of three column partials where
  // the CTAs on one SM fit in its 512 TMEM columns (16 channels); else four single buffers where
  // they fit (32 channels, two CTAs per SM), else two buffers of three partials (64 channels)
  if (conv_tmem_cols(12, a.np) * per_sm <= 512) {
    la.nacc = 4;
    la.nsplit = 3;
  } else if (conv_tmem_cols(4, a.np) * per_sm <= 512 && per_sm > 1) {
    la.nacc = 4;
    la.nsplit = 1;
  } else {
    la.nacc = 2;
    la.nsplit = conv_tmem_cols(6, a.np) * per_sm <= 512 ? 3 : 1;
  }
  if (ctas_per_replica) *ctas_per_replica = 4 * cpr;  // statistics partials: one per epilogue warp
  return launch_pdl(conv_tc_kernel, dim3(cpr, a.G), dim3(cv::THREADS), smem, stream, la);
}

cudaError_t launch_wgrad_update(const WgradUpdateArgs& a, cudaStream_t stream) {
  static_assert(sizeof(WgradUpdateArgs) <= 4096, "kernel parameter size");
  if (a.nl < 1 || a.nl > kWgradMaxLayers) return cudaErrorInvalidValue;
  if (a.G <= 0) return cudaSuccess;
  if (a.Kd <= 0 || !a.sgd.w || (a.sgd.mom != 0.f && !a.sgd.u)) return cudaErrorInvalidValue;
  int64_t tiles = 0;
  for (int l = 0; l < a.nl; ++l) {
    const WgradUpdateLayer& ly = a.L[l];
    if (ly.M <= 0 || ly.N <= 0) return cudaErrorInvalidValue;
    // operand boxes as the kernel expects them (64-wide MN-major boxes, or full K-major tiles),
    // with the same layouts in every layer
    if (ly.A.mn_major ? ly.A.box_rows != 64 : ly.A.box_rows != BM) return cudaErrorInvalidValue;
    if (ly.B.mn_major ? ly.B.box_rows != 64 : ly.B.box_rows != wu::TN) return cudaErrorInvalidValue;
    if (ly.A.mn_major != a.L[0].A.mn_major || ly.B.mn_major != a.L[0].B.mn_major)
      return cudaErrorInvalidValue;
    tiles += (int64_t)((ly.N + wu::TN - 1) / wu::TN) * ((ly.M + BM - 1) / BM) * a.G;
  }
  if (tiles > 0x7fffffffLL) return cudaErrorInvalidValue;
  // averaging mode, or replica 0's parameters for all: a CTA per tile position (all G replicas
  // of it), at most one per SM
  const int64_t units = (a.avg || a.w_rep0) ? tiles / a.G : tiles;
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  constexpr size_t smem = sizeof(WuSmem) + 1024;
  static_assert(smem <= 232448, "shared memory per CTA");
  static int attr_dev = -1;
  if (attr_dev != dev) {
    e = cudaFuncSetAttribute(wgrad_update_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
    if (e != cudaSuccess) return e;
    attr_dev = dev;
  }
  const int grid = (int)std::min<int64_t>(units, sms);
  launch_pdl(wgrad_update_kernel, dim3(grid), dim3(wu::THREADS), smem, stream, a);
  return cudaGetLastError();
}

bool conv_tile_shape(int hout, int wout, int* rows, int* images) {
  if (wout < 1 || hout < 1 || wout > BM || BM % wout) return false;
  const int per_image = hout * wout;
  if (per_image >= BM) {
    if (per_image % BM) return false;
    *rows = BM / wout;
    *images = 1;
  } else {
    if (BM % per_image) return false;
    *rows = hout;
    *images = BM / per_image;
  }
  return true;
}

bool conv_strip_ok(int hout, int wout, int stride) {
  int rows = 0, images = 0;
  // the kernel-row offsets inside a box must be whole swizzle atoms (8 pixel rows of the
  // channel width): wout a multiple of 8
  return stride == 1 && conv_tile_shape(hout, wout, &rows, &images) && images == 1 &&
         wout % 8 == 0 && rows + 2 <= 256;
}

bool make_tma_map_conv(CUtensorMap* map, const void* base, int ck, int win, int hin, int B, int G,
                       int wout, int hout, int stride, bool strip) {
  std::call_once(g_encode_once, load_encode);
  int rows = 0, images = 0;
  if (!g_encode || (ck != 16 && ck != 32 && ck != 64) || (stride != 1 && stride != 2) ||
      !conv_tile_shape(hout, wout, &rows, &images) || (reinterpret_cast<uintptr_t>(base) & 15))
    return false;
  if (wout * stride > 256 || rows * stride > 256 || images > 256) return false;
  const uint64_t e = 2;
  cuuint64_t dims[5] = {(cuuint64_t)ck, (cuuint64_t)win, (cuuint64_t)hin, (cuuint64_t)B,
                        (cuuint64_t)G};
  cuuint64_t strides[4] = {(cuuint64_t)ck * e, (cuuint64_t)win * ck * e,
                           (cuuint64_t)hin * win * ck * e, (cuuint64_t)B * hin * win * ck * e};
  // the strip form's box has a halo row above and below
  if (strip && !conv_strip_ok(hout, wout, stride)) return false;
  const int box_rows = strip ? rows + 2 : rows * stride;
  cuuint32_t box[5] = {(cuuint32_t)ck, (cuuint32_t)(wout * stride), (cuuint32_t)box_rows,
                       (cuuint32_t)images, 1};
  cuuint32_t estr[5] = {1, (cuuint32_t)stride, (cuuint32_t)stride, 1, 1};
  const CUtensorMapSwizzle sw = ck == 64 ? CU_TENSOR_MAP_SWIZZLE_128B
                                         : (ck == 32 ? CU_TENSOR_MAP_SWIZZLE_64B
                                                     : CU_TENSOR_MAP_SWIZZLE_32B);
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void*>(base), dims,
                        strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, sw,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool conv_wgrad_tc_ok(int cin, int cout, int stride, int hin, int win, int hout, int wout) {
  if ((cin != 16 && cin != 32 && cin != 64) || cout < 16 || cout > 64 || cout % 16) return false;
  if ((stride != 1 && stride != 2) || wout < 1 || wout > cw::KB || cw::KB % wout) return false;
  if ((hout * wout) % cw::KB || win != wout * stride || hin != hout * stride) return false;
  return win <= 256 && cw_rows(stride, wout) <= 256;
}

// Buffers and CTAs per SM of a shape.  Two A tiles; the input ring gets the rest of the shared
// memory (deeper rings measured faster than more A tiles).  Two CTAs per SM whenever each still
// gets three input stages: a CTA's blocks pass through a chain of handshakes one after another,
// and a second CTA overlaps its chain with the first's.
static void conv_wgrad_plan(int cin, int stride, int win, int wout, int* na, int* ni, int* per_sm,
                            size_t* smem) {
  const int mt_n = (9 * cin + 127) / 128;
  const size_t bars = (2 * cw::MAX_NI + 2 * cw::MAX_NA + 1) * 8 + 16;
  const size_t stage = cw_halo_pitch(cin, stride, win, wout) + cw::kTileB;
  auto fixed = [&](int nA) { return 1024 + (size_t)nA * mt_n * cw::kTileA + bars; };
  auto stages = [&](int nA, size_t budget) {
    return budget > fixed(nA) ? (int)std::min<size_t>(cw::MAX_NI, (budget - fixed(nA)) / stage) : 0;
  };
  const int n2 = stages(2, cw::kTwoPerSm), n1 = stages(2, cw::kOnePerSm);
  const int n2s = stages(1, cw::kTwoPerSm);  // one A tile: builders and MMAs take turns
  *na = 2;
  if (n2 >= 3 || (n2 >= 2 && 2 * n2 >= n1)) {
    *ni = n2;
    *per_sm = 2;
  } else if (n2s >= 3) {
    *na = 1;
    *ni = n2s;
    *per_sm = 2;
  } else {
    *ni = n1;
    *per_sm = 1;
  }
  *smem = *ni >= 2 ? fixed(*na) + (size_t)*ni * stage : 0;
}

int conv_wgrad_ctas(int cin, int stride, int wout, int G, int64_t P) {
  int na = 0, ni = 0, per_sm = 1;
  size_t smem = 0;
  conv_wgrad_plan(cin, stride, wout * stride, wout, &na, &ni, &per_sm, &smem);
  const int64_t blocks = P / cw::KB;
  return (int)std::max<int64_t>(1, std::min<int64_t>(blocks, (int64_t)kNumSMs * per_sm / std::max(G, 1)));
}

bool make_tma_map_halo(CUtensorMap* map, const void* base, int cin, int win, int hin, int B, int G,
                       int stride, int wout) {
  std::call_once(g_encode_once, load_encode);
  if (!g_encode || (cin != 16 && cin != 32 && cin != 64) || (reinterpret_cast<uintptr_t>(base) & 15))
    return false;
  const int rh = cw_rows(stride, wout);
  if (win > 256 || rh > 256) return false;
  const uint64_t e = 2;
  cuuint64_t dims[5] = {(cuuint64_t)cin, (cuuint64_t)win, (cuuint64_t)hin, (cuuint64_t)B,
                        (cuuint64_t)G};
  cuuint64_t strides[4] = {(cuuint64_t)cin * e, (cuuint64_t)win * cin * e,
                           (cuuint64_t)hin * win * cin * e, (cuuint64_t)B * hin * win * cin * e};
  cuuint32_t box[5] = {(cuuint32_t)cin, (cuuint32_t)win, (cuuint32_t)rh, 1, 1};
  cuuint32_t estr[5] = {1, 1, 1, 1, 1};
  // each pixel's channels are one 32 / 64 / 128-byte row, swizzled at that width so that the
  // builders' reads of neighbouring pixels spread over the banks
  const CUtensorMapSwizzle sw = cin == 64 ? CU_TENSOR_MAP_SWIZZLE_128B
                                          : (cin == 32 ? CU_TENSOR_MAP_SWIZZLE_64B
                                                       : CU_TENSOR_MAP_SWIZZLE_32B);
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void*>(base), dims,
                        strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, sw,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

cudaError_t launch_conv_wgrad_tc(const ConvWgradArgs& a, cudaStream_t stream) {
  if (a.P <= 0 || a.G <= 0) return cudaSuccess;
  if (!conv_wgrad_tc_ok(a.cin, a.cout, a.stride, a.hin, a.win, a.hout, a.wout) || !a.part ||
      a.P % cw::KB || a.P % (a.hout * a.wout) || a.cpr < 1 || a.cpr > a.P / cw::KB ||
      a.G > 65535 || (9 * a.cin + 127) / 128 > cw::MAX_MT)
    return cudaErrorInvalidValue;
  int na = 0, ni = 0, per_sm = 1;
  size_t smem = 0;
  conv_wgrad_plan(a.cin, a.stride, a.win, a.wout, &na, &ni, &per_sm, &smem);
  if (ni < 2 || ni > cw::MAX_NI || na < 1 || na > cw::MAX_NA || smem > 232448 ||
      (a.nb != 16 && a.nb != 32 && a.nb != 64) || a.nb < a.cout)
    return cudaErrorInvalidValue;
  ConvWgradArgs la = a;
  la.ni = ni;
  la.na = na;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  static int attr_dev = -1;
  if (attr_dev != dev) {
    e = cudaFuncSetAttribute(conv_wgrad_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             232448);
    if (e != cudaSuccess) return e;
    attr_dev = dev;
  }
  launch_pdl(conv_wgrad_tc_kernel, dim3(a.cpr, a.G), dim3(cw::THREADS), smem, stream, la);
  return cudaGetLastError();
}

int tc_tile_n(int Kd) { return (Kd + BK - 1) / BK <= 2 ? 128 : 64; }

int tc_valid_splits(int Kd, int want) {
  const int nk_all = (Kd + BK - 1) / BK;
  if (want < 1) want = 1;
  if (want > nk_all) want = nk_all;
  const int per = (nk_all + want - 1) / want;
  return (nk_all + per - 1) / per;  // every split gets at least one k-block
}

namespace {
bool gemm_pt_off() {
  static const bool off = [] {
    const char* e = std::getenv("LSGD_GEMM_ONE_TILE");
    return e && e[0] == '1';
  }();
  return off;
}

cudaError_t launch_pt(const TcGemmArgs& a, cudaStream_t stream) {
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  constexpr size_t smem = sizeof(PtSmem) + 1024;
  static_assert(smem <= 232448, "shared memory per CTA");
  static int attr_dev = -1;
  if (attr_dev != dev) {
    e = cudaFuncSetAttribute(gemm_pt_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    attr_dev = dev;
  }
  const int64_t tiles = (int64_t)((a.N + pt::PBN - 1) / pt::PBN) * ((a.M + BM - 1) / BM) * a.G;
  if (tiles > 0x7fffffffLL) return cudaErrorInvalidValue;
  const int grid = (int)std::min<int64_t>(tiles, sms);
  launch_pdl(gemm_pt_kernel, dim3(grid), dim3(pt::THREADS), smem, stream, a);
  return cudaGetLastError();
}
}  // namespace

cudaError_t launch_gemm_tc(const TcGemmArgs& a, cudaStream_t stream) {
  if (a.M <= 0 || a.N <= 0 || a.G <= 0) return cudaSuccess;
  if (a.Kd <= 0 || a.G > 65535) return cudaErrorInvalidValue;
  // The TMA boxes must deliver exactly the tiles the kernel expects (expect-tx byte counts and
  // shared-memory extents depend on it).
  const int bn = tc_tile_n(a.Kd);
  if (a.A.mn_major ? a.A.box_rows != 64 : a.A.box_rows != BM) return cudaErrorInvalidValue;
  if (a.B.mn_major ? a.B.box_rows != 64 : a.B.box_rows != bn) return cudaErrorInvalidValue;
  if ((a.epi == EPI_BIAS || a.epi == EPI_BIAS_RELU) && !a.bias) return cudaErrorInvalidValue;
  if (a.epi == EPI_MASK && !a.mask) return cudaErrorInvalidValue;
  if (!a.C) return cudaErrorInvalidValue;
  if (a.conv) {
    // K-major tap slices of cv_ck channels on both sides; 64-wide N tiles, four stages, no split
    int rows = 0, images = 0;
    if ((a.cv_ck != 16 && a.cv_ck != 32 && a.cv_ck != 64) || (a.cv_stride != 1 && a.cv_stride != 2) ||
        !conv_tile_shape(a.cv_hout, a.cv_wout, &rows, &images) || a.splits > 1 ||
        a.A.mn_major || a.B.mn_major || a.bias_colsum)
      return cudaErrorInvalidValue;
    if (a.M % (a.cv_hout * a.cv_wout)) return cudaErrorInvalidValue;  // whole images
    dim3 gridc((a.N + 63) / 64, (a.M + BM - 1) / BM, a.G);
    if (gridc.y > 65535) return cudaErrorInvalidValue;
    return launch_cfg<64, 4>(a, gridc, stream);
  }
  // the bias column sums need the whole mini-batch in one tile, and the masked data gradient
  if (a.bias_colsum && (a.M > BM || a.epi != EPI_MASK || (!a.bsgd.w && !a.bias_grad)))
    return cudaErrorInvalidValue;
  const int splits = a.splits > 1 ? a.splits : 1;
  if (splits > 1) {
    const int nk_all = (a.Kd + BK - 1) / BK, per = (nk_all + splits - 1) / splits;
    if (a.epi != EPI_STORE || (int64_t)(splits - 1) * per >= nk_all) return cudaErrorInvalidValue;
    if ((int64_t)a.G * splits > 65535) return cudaErrorInvalidValue;
  }
  constexpr int BN = 128;
  dim3 grid((a.N + BN - 1) / BN, (a.M + BM - 1) / BM, a.G * splits);
  if (grid.y > 65535) return cudaErrorInvalidValue;
  static_assert(BM == kTcTileM, "tile height");
  // Short reductions (the weight gradient's k = B_loc) need only two stages; the smaller shared
  // footprint lets three CTAs share an SM so one CTA's epilogue overlaps the others' loads.
  if ((a.Kd + BK - 1) / BK <= 2) return launch_cfg<BN, 2>(a, grid, stream);
  // Wide products (at least 2048 output columns, no split): the persistent kernel -- the forward
  // (K-major weights) and, since its epilogue prefetches the tile's ReLU mask, the data gradient
  // (MN-major weights).  Narrower layers give it too few 128 x 256 tiles to fill the SMs
  // (measured: MLP 3072-4096x3-100 forward 0.36 -> 0.27 ms per step, backward 0.333 -> 0.322 ms;
  // MLP 3072-1024-1024-10 0.29 -> 0.35 ms per step, so it stays on the one-tile kernel).
  if (splits == 1 && a.N >= 2048 && a.B.box_rows == 64 && !gemm_pt_off())
    return launch_pt(a, stream);
  // Other long reductions: 64-wide N tiles with four stages (96 KB) so two CTAs share an SM and
  // twice as many tiles stream weights at once.
  constexpr int BN2 = 64;
  dim3 grid2((a.N + BN2 - 1) / BN2, (a.M + BM - 1) / BM, a.G * splits);
  return launch_cfg<BN2, 4>(a, grid2, stream);
}

}  // namespace lsgd
