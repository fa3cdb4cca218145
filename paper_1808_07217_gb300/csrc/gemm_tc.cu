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
#include <cudaTypedefs.h>

#include <mutex>

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

// Fetch a tensor tile into L2 only (no shared memory, no completion tracking).
__device__ __forceinline__ void tma_prefetch_l2_3d(const CUtensorMap* map, int x, int y, int z) {
  asm volatile("cp.async.bulk.prefetch.tensor.3d.L2.global.tile [%0, {%1, %2, %3}];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(x), "r"(y), "r"(z)
               : "memory");
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

// The local update on four consecutive parameters (fused weight-gradient epilogue).
__device__ __forceinline__ void sgd4(float4& w, float4& u, const float4 g, const SgdParams& sp) {
  const bool sg = sp.sign != 0;
  if (sp.mom == 0.f) {
    sgd_elem<false, false>(w.x, u.x, g.x, sp.lr, 0.f, sp.wd, sg);
    sgd_elem<false, false>(w.y, u.y, g.y, sp.lr, 0.f, sp.wd, sg);
    sgd_elem<false, false>(w.z, u.z, g.z, sp.lr, 0.f, sp.wd, sg);
    sgd_elem<false, false>(w.w, u.w, g.w, sp.lr, 0.f, sp.wd, sg);
  } else if (sp.nesterov) {
    sgd_elem<true, true>(w.x, u.x, g.x, sp.lr, sp.mom, sp.wd, sg);
    sgd_elem<true, true>(w.y, u.y, g.y, sp.lr, sp.mom, sp.wd, sg);
    sgd_elem<true, true>(w.z, u.z, g.z, sp.lr, sp.mom, sp.wd, sg);
    sgd_elem<true, true>(w.w, u.w, g.w, sp.lr, sp.mom, sp.wd, sg);
  } else {
    sgd_elem<true, false>(w.x, u.x, g.x, sp.lr, sp.mom, sp.wd, sg);
    sgd_elem<true, false>(w.y, u.y, g.y, sp.lr, sp.mom, sp.wd, sg);
    sgd_elem<true, false>(w.z, u.z, g.z, sp.lr, sp.mom, sp.wd, sg);
    sgd_elem<true, false>(w.w, u.w, g.w, sp.lr, sp.mom, sp.wd, sg);
  }
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

template <int BN, int STAGES>
__global__ void __launch_bounds__(128, 1) gemm_tc_kernel(const __grid_constant__ TcGemmArgs args) {
  extern __shared__ uint8_t smem_raw[];
  Smem<BN, STAGES>& sm = *reinterpret_cast<Smem<BN, STAGES>*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int splits = args.splits > 1 ? args.splits : 1;
  const int n0 = blockIdx.x * BN, m0 = blockIdx.y * BM, g = blockIdx.z / splits;
  const int split = blockIdx.z % splits;
  const int nk_all = (args.Kd + BK - 1) / BK;
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

  bool ok = true;
  if (warp == 0 && lane == 0) {
    // ---------------- TMA producer ----------------
    if (args.epi == EPI_SGD && args.have_wu_maps) {
      // the epilogue reads this tile's parameters and momentum: start them towards L2 now
#pragma unroll
      for (int i = 0; i < BN / 64; ++i) {
        tma_prefetch_l2_3d(&args.wmap, n0 + 64 * i, m0, g);
        if (args.sgd.u) tma_prefetch_l2_3d(&args.umap, n0 + 64 * i, m0, g);
      }
    }
    int issued = 0;
    for (int kb = 0; kb < nk && ok; ++kb) {
      const int s = kb % STAGES;
      const uint32_t ph = (kb / STAGES) & 1;
      if (!mbar_wait(&sm.empty[s], ph ^ 1)) {
        ok = false;
        break;
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
      if (!b_mn) {
        tma_load_3d(sm.b[s], &args.B.map, &sm.full[s], k0, n0, g);
      } else {
#pragma unroll
        for (int i = 0; i < BN / 64; ++i)
          tma_load_3d(sm.b[s] + i * 64 * BK * 2, &args.B.map, &sm.full[s], n0 + 64 * i, k0, g);
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
  }
  __syncwarp();

  // ---------------- epilogue (all 4 warps) ----------------
  // The stage buffers are free once the accumulator is complete (every MMA has read its
  // operands).  The tile leaves TMEM in 64-column chunks: each thread takes its row's 64 fp32
  // values (bias / ReLU applied), writes them to a padded shared-memory staging tile, and the CTA
  // then stores the chunk row-contiguously (a warp writes two 256-byte row segments per
  // instruction), applying the ReLU mask from a coalesced read of the stored activation.
  const bool have_acc = mbar_wait(&sm.accum, 0);
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  if (have_acc) {
    constexpr int CW = 64, PITCH = CW + 4;  // staged chunk width and row pitch (floats)
    float* stg = reinterpret_cast<float*>(sm.a[0]);
    const int r = warp * 32 + lane;  // tile row owned in the TMEM phase
    const float* bias = args.bias ? args.bias + (int64_t)g * args.bias_gs : nullptr;
    const int epi = args.epi;
    for (int cc = 0; cc < BN; cc += CW) {
      if (n0 + cc >= args.N) break;  // block-uniform
#pragma unroll
      for (int q = 0; q < CW / 16; ++q) {
        float v[16];
        tmem_ld16(tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)(cc + 16 * q), v);
        if (epi == EPI_BIAS || epi == EPI_BIAS_RELU) {
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const int n = n0 + cc + 16 * q + i;
            float x = v[i] + (n < args.N ? __ldg(bias + n) : 0.f);
            v[i] = (epi == EPI_BIAS_RELU) ? fmaxf(x, 0.f) : x;
          }
        }
        float4* dst = reinterpret_cast<float4*>(stg + r * PITCH + 16 * q);
#pragma unroll
        for (int i = 0; i < 4; ++i) dst[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
      }
      asm volatile("bar.sync 1, 128;" ::: "memory");
      // copy-out: item = (row, 4-column group), 16 groups per 64-column row.  Each thread takes
      // UNR items at a time and issues all their global loads (mask, or w and u) before any
      // arithmetic, so several hundred bytes per thread are in flight.
      constexpr int UNR = 8, ITEMS = BM * (CW / 4);
      for (int base = threadIdx.x; base < ITEMS; base += 128 * UNR) {
        float4 x[UNR], a0[UNR], a1[UNR];
        int64_t off[UNR];
        int nn[UNR];
        bool ok[UNR];
#pragma unroll
        for (int q = 0; q < UNR; ++q) {
          const int it = base + q * 128;
          const int row = it / (CW / 4), grp = it % (CW / 4);
          const int m = m0 + row, n = n0 + cc + grp * 4;
          ok[q] = it < ITEMS && m < args.M && n < args.N;
          nn[q] = n;
          off[q] = c_base + (int64_t)m * args.c_rs + n;
          a0[q] = make_float4(0.f, 0.f, 0.f, 0.f);
          a1[q] = a0[q];
          if (!ok[q]) continue;
          x[q] = *reinterpret_cast<const float4*>(stg + row * PITCH + grp * 4);
          const bool full4 = n + 4 <= args.N;
          if (epi == EPI_MASK) {
            const int64_t moff = (int64_t)g * args.mask_gs + (int64_t)m * args.mask_rs + n;
            if (args.mask_bf16) {
              const uint16_t* mp = reinterpret_cast<const uint16_t*>(args.mask) + moff;
              if (full4 && ((reinterpret_cast<uintptr_t>(mp) & 7) == 0)) {
                const uint2 u = __ldg(reinterpret_cast<const uint2*>(mp));
                a0[q] = make_float4(bf2f((uint16_t)(u.x & 0xffff)), bf2f((uint16_t)(u.x >> 16)),
                                    bf2f((uint16_t)(u.y & 0xffff)), bf2f((uint16_t)(u.y >> 16)));
              } else {
                float t[4] = {0.f, 0.f, 0.f, 0.f};
                for (int i = 0; i < 4 && n + i < args.N; ++i) t[i] = bf2f(mp[i]);
                a0[q] = make_float4(t[0], t[1], t[2], t[3]);
              }
            } else {
              const float* mp = reinterpret_cast<const float*>(args.mask) + moff;
              float t[4] = {0.f, 0.f, 0.f, 0.f};
              for (int i = 0; i < 4 && n + i < args.N; ++i) t[i] = mp[i];
              a0[q] = make_float4(t[0], t[1], t[2], t[3]);
            }
          } else if (epi == EPI_SGD) {
            const float* wp = args.sgd.w + off[q];
            const float* up = args.sgd.u ? args.sgd.u + off[q] : nullptr;
            if (full4 && ((reinterpret_cast<uintptr_t>(wp) & 15) == 0) &&
                ((reinterpret_cast<uintptr_t>(up) & 15) == 0)) {
              a0[q] = __ldcs(reinterpret_cast<const float4*>(wp));
              if (up) a1[q] = __ldcs(reinterpret_cast<const float4*>(up));
            } else {
              float t[4] = {0.f, 0.f, 0.f, 0.f}, v[4] = {0.f, 0.f, 0.f, 0.f};
              for (int i = 0; i < 4 && n + i < args.N; ++i) {
                t[i] = wp[i];
                if (up) v[i] = up[i];
              }
              a0[q] = make_float4(t[0], t[1], t[2], t[3]);
              a1[q] = make_float4(v[0], v[1], v[2], v[3]);
            }
          }
        }
#pragma unroll
        for (int q = 0; q < UNR; ++q) {
          if (!ok[q]) continue;
          const int n = nn[q];
          const bool full4 = n + 4 <= args.N;
          float4 v = x[q];
          if (epi == EPI_MASK) {
            v.x = a0[q].x > 0.f ? v.x : 0.f;
            v.y = a0[q].y > 0.f ? v.y : 0.f;
            v.z = a0[q].z > 0.f ? v.z : 0.f;
            v.w = a0[q].w > 0.f ? v.w : 0.f;
          }
          if (epi == EPI_SGD) {
            const SgdParams& sp = args.sgd;
            float4 wv = a0[q], uv = a1[q];
            sgd4(wv, uv, v, sp);
            float* wp = sp.w + off[q];
            float* up = sp.u ? sp.u + off[q] : nullptr;
            uint16_t* bp = sp.wb ? sp.wb + off[q] : nullptr;
            if (full4 && ((reinterpret_cast<uintptr_t>(wp) & 15) == 0) &&
                ((reinterpret_cast<uintptr_t>(up) & 15) == 0) &&
                ((reinterpret_cast<uintptr_t>(bp) & 7) == 0)) {
              __stcs(reinterpret_cast<float4*>(wp), wv);
              if (up) __stcs(reinterpret_cast<float4*>(up), uv);
              if (bp) {
                uint2 o;
                o.x = (uint32_t)f2bf(wv.x) | ((uint32_t)f2bf(wv.y) << 16);
                o.y = (uint32_t)f2bf(wv.z) | ((uint32_t)f2bf(wv.w) << 16);
                __stcs(reinterpret_cast<uint2*>(bp), o);
              }
            } else {
              const float ws[4] = {wv.x, wv.y, wv.z, wv.w}, us[4] = {uv.x, uv.y, uv.z, uv.w};
              for (int i = 0; i < 4 && n + i < args.N; ++i) {
                wp[i] = ws[i];
                if (up) up[i] = us[i];
                if (bp) bp[i] = f2bf(ws[i]);
              }
            }
            continue;
          }
          if (args.c_bf16) {
            uint16_t* out = reinterpret_cast<uint16_t*>(args.C) + off[q];
            if (full4 && ((reinterpret_cast<uintptr_t>(out) & 7) == 0)) {
              uint2 o;
              o.x = (uint32_t)f2bf(v.x) | ((uint32_t)f2bf(v.y) << 16);
              o.y = (uint32_t)f2bf(v.z) | ((uint32_t)f2bf(v.w) << 16);
              *reinterpret_cast<uint2*>(out) = o;
            } else {
              const float xs[4] = {v.x, v.y, v.z, v.w};
              for (int i = 0; i < 4 && n + i < args.N; ++i) out[i] = f2bf(xs[i]);
            }
          } else {
            float* out = reinterpret_cast<float*>(args.C) + off[q];
            if (full4 && ((reinterpret_cast<uintptr_t>(out) & 15) == 0)) {
              *reinterpret_cast<float4*>(out) = v;
            } else {
              const float xs[4] = {v.x, v.y, v.z, v.w};
              for (int i = 0; i < 4 && n + i < args.N; ++i) out[i] = xs[i];
            }
          }
        }
      }
      asm volatile("bar.sync 1, 128;" ::: "memory");
    }
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (warp == 2) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"((uint32_t)BN)
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
  gemm_tc_kernel<BN, STAGES><<<grid, 128, smem, stream>>>(a);
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

int tc_tile_n(int Kd) { return (Kd + BK - 1) / BK <= 2 ? 128 : 64; }

int tc_valid_splits(int Kd, int want) {
  const int nk_all = (Kd + BK - 1) / BK;
  if (want < 1) want = 1;
  if (want > nk_all) want = nk_all;
  const int per = (nk_all + want - 1) / want;
  return (nk_all + per - 1) / per;  // every split gets at least one k-block
}

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
  if (a.epi == EPI_SGD && (!a.sgd.w || (a.sgd.mom != 0.f && !a.sgd.u))) return cudaErrorInvalidValue;
  if (a.epi != EPI_SGD && !a.C) return cudaErrorInvalidValue;
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
  // Long reductions (forward, data gradient): 64-wide N tiles with four stages (96 KB) so two
  // CTAs share an SM and twice as many tiles stream weights at once.
  constexpr int BN2 = 64;
  dim3 grid2((a.N + BN2 - 1) / BN2, (a.M + BM - 1) / BM, a.G * splits);
  return launch_cfg<BN2, 4>(a, grid2, stream);
}

}  // namespace lsgd
