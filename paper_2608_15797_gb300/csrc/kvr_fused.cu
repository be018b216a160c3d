// kvr_fused.cu -- the fused steady-state decode step for bf16, head_dim 128,
// G <= 8 and at most 128 live rows per unit: append + Attn(q_t, C) (Eq. 1)
// + accumulated-attention update (Sec. 2.1) + TopB eviction of the single
// surplus row (Eq. 1 with the Sec. 4.1 window) + in-place compaction, in one
// pass over K and V.
//
// Design (GB300, sm_103a):
//  - Persistent CTAs, one per SM.  Each CTA owns a ring of shared-memory
//    stages; a producer warp fills a stage with one unit's K and V (two
//    128B-swizzled TMA boxes each: columns 0-63 and 64-127, all rows of the
//    unit), its G query rows, the new k/v row, scores, positions and state,
//    all completing on the stage's mbarrier.  Four consumer warps each
//    process whole units, one warp per unit.
//  - QK^T and PV run on warp-level bf16 tensor-core MMAs (m16n8k16, fp32
//    accumulate): K rows are the M side, the <= 8 query heads of the group
//    the N side.  The probability tile leaves the QK accumulators in
//    registers and becomes the PV B operand through movmatrix (an 8x8
//    transpose), so P never touches memory.  Softmax and score reductions
//    are warp shuffles.
//  - The new row is inserted into the staged tile, so K and V are read once
//    from HBM and nothing is re-read for the scores.  Exactly one row is
//    evicted (warp argmin of the (score, -position) key over non-window
//    rows) and the new row is written straight into the freed slot: the
//    compaction moves no other row.
//  - Every wait on an mbarrier is bounded (about 2 s); on timeout the kernel
//    sets ERR_TIMEOUT in the device error word and drains its own copies.
#include <cuda.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "kvr_internal.h"

namespace kvr {
namespace {

constexpr int kMaxStages = 8;
constexpr int kMaxGroups = 4;      // units in flight on the consumer side
constexpr int kMaxGroupWarps = 8;  // warps sharing one unit
constexpr int kMaxThreads = 544;   // 16 consumer warps + the producer
constexpr int kXsWords = 20;       // exchange words per warp of a group
constexpr int kQPitch = 272;  // bytes per staged query row (256 + 16 padding)
constexpr uint64_t kWaitNs = 2000000000ull;

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count)
               : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// Bounded wait; false on timeout or when another warp raised `abort`.
__device__ bool mbar_wait(uint32_t bar, uint32_t parity,
                          volatile int *abort) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (*abort || global_ns() - t0 > kWaitNs) return false;
  }
  return true;
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void fence_proxy_async() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *map,
                                            int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_"
      "tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}
__device__ __forceinline__ void bulk_load(uint32_t dst, const void *src,
                                          uint32_t bytes, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], "
      "[%1], %2, [%3];" ::"r"(dst),
      "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t &r0,
                                        uint32_t &r1, uint32_t &r2,
                                        uint32_t &r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t &r0,
                                          uint32_t &r1, uint32_t &r2,
                                          uint32_t &r3) {
  asm volatile(
      "ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
      : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
      : "r"(addr));
}
__device__ __forceinline__ void mma_bf16(float (&d)[4], uint32_t a0,
                                         uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, "
      "{%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t movm_t(uint32_t x) {
  uint32_t y;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;"
               : "=r"(y)
               : "r"(x));
  return y;
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t *>(&v);
}

__device__ __forceinline__ void group_bar(int id, int threads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

// Byte offsets inside one stage of R staged rows.
struct StageLayout {
  uint32_t k0, k1, v0, v1, q, kn, vn, sc, ps, st, xs, bytes;
  __host__ __device__ explicit StageLayout(int R) {
    k0 = 0;
    k1 = k0 + R * 128;
    v0 = k1 + R * 128;
    v1 = v0 + R * 128;
    q = v1 + R * 128;
    kn = q + 8 * kQPitch;
    vn = kn + 256;
    sc = vn + 256;
    ps = sc + 4 * R;
    st = ps + 4 * R;
    xs = st + 16;  // group exchange: kXsWords words per warp
    bytes = ((xs + 4 * kXsWords * kMaxGroupWarps) + 1023) / 1024 * 1024;
  }
};

struct UnitIdx {
  int h, lr, sq;
  size_t ug;    // cache unit
  size_t krow;  // row of this unit in the call's [S][nl][H] inputs
};

__device__ __forceinline__ UnitIdx unit_idx(const FusedParams &p, int idx) {
  UnitIdx x;
  x.h = idx % p.c.H;
  x.lr = (idx / p.c.H) % p.nl;
  x.sq = idx / (p.c.H * p.nl);
  x.ug = ((size_t)x.sq * p.c.L + p.lb + x.lr) * p.c.H + x.h;
  x.krow = ((size_t)x.sq * p.nl + x.lr) * p.c.H + x.h;
  return x;
}

// Producer: enqueue every copy of one unit into a stage.  K and V come as
// two 128B-swizzled boxes of Rb rows each (columns 0-63, 64-127).
__device__ void issue_unit(const FusedParams &p, const CUtensorMap *tmK,
                           const CUtensorMap *tmV, unsigned char *stage,
                           uint32_t bar, int idx) {
  const StageLayout L(p.R);
  const UnitIdx x = unit_idx(p, idx);
  const int G = p.c.G;
  const uint32_t s0 = smem_u32(stage);
  const uint32_t tx = 4u * p.Rb * 128u + (uint32_t)G * 256u + 512u +
                      8u * p.Rb + 16u;
  mbar_expect_tx(bar, tx);
  const int row0 = (int)(x.ug * (size_t)p.c.cap);
  tma_load_2d(s0 + L.k0, tmK, 0, row0, bar);
  tma_load_2d(s0 + L.k1, tmK, 64, row0, bar);
  tma_load_2d(s0 + L.v0, tmV, 0, row0, bar);
  tma_load_2d(s0 + L.v1, tmV, 64, row0, bar);
  const __nv_bfloat16 *q = p.q + x.krow * G * 128;
  for (int g = 0; g < G; ++g)
    bulk_load(s0 + L.q + g * kQPitch, q + g * 128, 256, bar);
  bulk_load(s0 + L.kn, p.k_new + x.krow * 128, 256, bar);
  bulk_load(s0 + L.vn, p.v_new + x.krow * 128, 256, bar);
  bulk_load(s0 + L.sc, p.c.score + x.ug * p.c.sstride, 4u * p.Rb, bar);
  bulk_load(s0 + L.ps, p.c.pos + x.ug * p.c.sstride, 4u * p.Rb, bar);
  bulk_load(s0 + L.st, p.c.state + x.ug * 4, 16, bar);
}

// One group of U warps computes one unit held in a stage.  The unit has
// T = R / 16 row tiles; warp w of the group owns tiles w, w + U, ...
// Exchange words per warp (XS): [0,8) column max, [8,16) column sum,
// [16,18) argmin key, 18 argmin row, 19 wait flag.
template <int T, int U, bool kOutBf16>
__device__ void process_unit(const FusedParams &p, unsigned char *stage,
                             int idx, int w, int lane, int bar_id) {
  constexpr int TW = (T + U - 1) / U;  // tiles per warp (at most)
  constexpr int R = 16 * T;
  constexpr int GT = 32 * U;           // threads of the group
  const StageLayout L(R);
  const UnitIdx x = unit_idx(p, idx);
  const int G = p.c.G;
  const int gt = w * 32 + lane;
  unsigned char *K0 = stage + L.k0, *K1 = stage + L.k1;
  unsigned char *V0 = stage + L.v0, *V1 = stage + L.v1;
  const unsigned char *KN = stage + L.kn, *VN = stage + L.vn;
  float *SC = reinterpret_cast<float *>(stage + L.sc);
  const int32_t *PS = reinterpret_cast<const int32_t *>(stage + L.ps);
  const int32_t *ST = reinterpret_cast<const int32_t *>(stage + L.st);
  float *XS = reinterpret_cast<float *>(stage + L.xs);
  const int m = ST[0], t = ST[1], n = m + 1;
  if (m < 0 || n > R) {  // same decision in every warp of the group
    if (gt == 0) atomicOr(p.c.err, ERR_LENGTH);
    return;
  }

  // 1. Insert the new row as logical row m (swizzled like the TMA boxes)
  //    and zero V beyond it, so padded rows contribute 0, not NaN.
  if (w == 0) {
    const int chunk = lane & 15, half = chunk >> 3, cc = chunk & 7;
    const uint32_t off = m * 128 + ((cc ^ (m & 7)) << 4);
    unsigned char *dst = lane < 16 ? (half ? K1 : K0) : (half ? V1 : V0);
    const unsigned char *src = lane < 16 ? KN : VN;
    *reinterpret_cast<int4 *>(dst + off) =
        *reinterpret_cast<const int4 *>(src + chunk * 16);
  }
  for (int i = gt; i < (R - m - 1) * 16; i += GT) {
    const int r = m + 1 + (i >> 4), c16 = i & 15;
    *reinterpret_cast<int4 *>((c16 < 8 ? V0 : V1) + r * 128 + (c16 & 7) * 16) =
        make_int4(0, 0, 0, 0);
  }
  group_bar(bar_id, GT);

  // 2. Query heads as the MMA B operand (k = head dim, n = query head).
  uint32_t qb[8][2];
  {
    const uint32_t qa = smem_u32(stage + L.q) + (lane & 7) * kQPitch +
                        (lane >> 3) * 16;
#pragma unroll
    for (int i = 0; i < 4; ++i)
      ldsm_x4(qa + i * 64, qb[2 * i][0], qb[2 * i][1], qb[2 * i + 1][0],
              qb[2 * i + 1][1]);
  }

  // 3. Logits of the owned tiles: m16n8 per 16 rows, 8 k-steps.
  float acc[TW][4];
#pragma unroll
  for (int j = 0; j < TW; ++j) {
    acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;
    const int tt = w + j * U;
    if (tt < T) {
      const int row = tt * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
      const uint32_t b0 = smem_u32(K0) + row * 128, b1 = smem_u32(K1) + row * 128;
#pragma unroll
      for (int ks = 0; ks < 8; ++ks) {
        const int cc = ((ks & 3) << 1) + (lane >> 4);
        const uint32_t addr = (ks >> 2 ? b1 : b0) + ((cc ^ (row & 7)) << 4);
        uint32_t a0, a1, a2, a3;
        ldsm_x4(addr, a0, a1, a2, a3);
        mma_bf16(acc[j], a0, a1, a2, a3, qb[ks][0], qb[ks][1]);
      }
    }
  }

  // 4. Softmax per query head: this lane holds columns c2 and c2 + 1.
  const int r0 = lane >> 2, c2 = (lane & 3) * 2;
  float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
  for (int j = 0; j < TW; ++j) {
    const int ra = (w + j * U) * 16 + r0, rb = ra + 8;  // rows >= n masked
    acc[j][0] = ra < n ? acc[j][0] * p.scale_log2e : -INFINITY;
    acc[j][1] = ra < n ? acc[j][1] * p.scale_log2e : -INFINITY;
    acc[j][2] = rb < n ? acc[j][2] * p.scale_log2e : -INFINITY;
    acc[j][3] = rb < n ? acc[j][3] * p.scale_log2e : -INFINITY;
    mx0 = fmaxf(mx0, fmaxf(acc[j][0], acc[j][2]));
    mx1 = fmaxf(mx1, fmaxf(acc[j][1], acc[j][3]));
  }
#pragma unroll
  for (int o = 4; o < 32; o <<= 1) {
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, o));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, o));
  }
  if (U > 1) {
    if (lane < 4) {
      XS[w * kXsWords + c2] = mx0;
      XS[w * kXsWords + c2 + 1] = mx1;
    }
    group_bar(bar_id, GT);
#pragma unroll
    for (int v = 0; v < U; ++v) {
      mx0 = fmaxf(mx0, XS[v * kXsWords + c2]);
      mx1 = fmaxf(mx1, XS[v * kXsWords + c2 + 1]);
    }
  }
  float z0 = 0.f, z1 = 0.f;
#pragma unroll
  for (int j = 0; j < TW; ++j) {
    acc[j][0] = exp2f(acc[j][0] - mx0);
    acc[j][1] = exp2f(acc[j][1] - mx1);
    acc[j][2] = exp2f(acc[j][2] - mx0);
    acc[j][3] = exp2f(acc[j][3] - mx1);
    z0 += acc[j][0] + acc[j][2];
    z1 += acc[j][1] + acc[j][3];
  }
#pragma unroll
  for (int o = 4; o < 32; o <<= 1) {
    z0 += __shfl_xor_sync(0xffffffffu, z0, o);
    z1 += __shfl_xor_sync(0xffffffffu, z1, o);
  }
  if (U > 1) {
    if (lane < 4) {
      XS[w * kXsWords + 8 + c2] = z0;
      XS[w * kXsWords + 8 + c2 + 1] = z1;
    }
    group_bar(bar_id, GT);
    z0 = z1 = 0.f;
#pragma unroll
    for (int v = 0; v < U; ++v) {
      z0 += XS[v * kXsWords + 8 + c2];
      z1 += XS[v * kXsWords + 8 + c2 + 1];
    }
  }
  if (gt == 0 && (!(z0 >= 1.f) || !(z0 < INFINITY)))
    atomicOr(p.c.err, ERR_NONFINITE);
  const float i0 = 1.f / z0, i1 = 1.f / z1;

  // 5. Accumulated attention: score += mean over the G heads (staged copy;
  //    every row belongs to exactly one warp).
  const bool g0 = c2 < G, g1 = c2 + 1 < G;
#pragma unroll
  for (int j = 0; j < TW; ++j) {
    acc[j][0] *= i0;
    acc[j][2] *= i0;
    acc[j][1] *= i1;
    acc[j][3] *= i1;
    float sa = (g0 ? acc[j][0] : 0.f) + (g1 ? acc[j][1] : 0.f);
    float sb = (g0 ? acc[j][2] : 0.f) + (g1 ? acc[j][3] : 0.f);
    sa += __shfl_xor_sync(0xffffffffu, sa, 1);
    sb += __shfl_xor_sync(0xffffffffu, sb, 1);
    sa += __shfl_xor_sync(0xffffffffu, sa, 2);
    sb += __shfl_xor_sync(0xffffffffu, sb, 2);
    if ((lane & 3) == 0) {
      const int ra = (w + j * U) * 16 + r0, rb = ra + 8;
      if (ra < m) SC[ra] += sa * p.inv_g;
      else if (ra == m) SC[ra] = sa * p.inv_g;
      if (rb < m) SC[rb] += sb * p.inv_g;
      else if (rb == m) SC[rb] = sb * p.inv_g;
    }
  }

  // 6. P as the PV B operand, split into two bf16 terms (hi + lo carries
  //    ~16 mantissa bits; a single bf16 P would cost up to 2^-9 relative
  //    per probability), each 8x8 block transposed in registers.
  uint32_t bp[TW][2], bl[TW][2];
#pragma unroll
  for (int j = 0; j < TW; ++j) {
    const uint32_t h0 = pack_bf16(acc[j][0], acc[j][1]);
    const uint32_t h1 = pack_bf16(acc[j][2], acc[j][3]);
    const __nv_bfloat162 hb0 = *reinterpret_cast<const __nv_bfloat162 *>(&h0);
    const __nv_bfloat162 hb1 = *reinterpret_cast<const __nv_bfloat162 *>(&h1);
    const uint32_t l0 = pack_bf16(acc[j][0] - __low2float(hb0),
                                  acc[j][1] - __high2float(hb0));
    const uint32_t l1 = pack_bf16(acc[j][2] - __low2float(hb1),
                                  acc[j][3] - __high2float(hb1));
    bp[j][0] = movm_t(h0);
    bp[j][1] = movm_t(h1);
    bl[j][0] = movm_t(l0);
    bl[j][1] = movm_t(l1);
  }

  // 7. Partial out^T = V^T P^T over the owned tiles: M = head dim (8 tiles
  //    of 16), K = rows, N = query heads.
  float o[8][4];
#pragma unroll
  for (int mt = 0; mt < 8; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
#pragma unroll
  for (int j = 0; j < TW; ++j) {
    const int tt = w + j * U;
    if (tt < T) {
      const int row = tt * 16 + (lane & 7) + ((lane >> 4) << 3);
      const uint32_t b0 = smem_u32(V0) + row * 128, b1 = smem_u32(V1) + row * 128;
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) {
        const int c16 = 2 * mt + ((lane >> 3) & 1);
        const uint32_t addr = (c16 >> 3 ? b1 : b0) + (((c16 & 7) ^ (row & 7)) << 4);
        uint32_t a0, a1, a2, a3;
        ldsm_x4_t(addr, a0, a1, a2, a3);
        mma_bf16(o[mt], a0, a1, a2, a3, bp[j][0], bp[j][1]);
        mma_bf16(o[mt], a0, a1, a2, a3, bl[j][0], bl[j][1]);
      }
    }
  }

  // 8. Sum the partials across the group (K area, free since every warp has
  //    passed the softmax exchange), stage the output rows in the V area
  //    (free once every warp has finished PV) and store them.
  constexpr int osz = kOutBf16 ? 2 : 4;
  const int pitch = 128 * osz + (G * (128 * osz + 16) <= 2 * R * 128 ? 16 : 0);
  unsigned char *OUT = V0;
  if (U > 1) {
    float *XO = reinterpret_cast<float *>(K0);
#pragma unroll
    for (int mt = 0; mt < 8; ++mt)
#pragma unroll
      for (int e = 0; e < 4; ++e) XO[((w * 8 + mt) * 4 + e) * 32 + lane] = o[mt][e];
    group_bar(bar_id, GT);
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) {
      if (mt % U == w) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          float sum = 0.f;
#pragma unroll
          for (int v = 0; v < U; ++v) sum += XO[((v * 8 + mt) * 4 + e) * 32 + lane];
          o[mt][e] = sum;
        }
      }
    }
  }
#pragma unroll
  for (int mt = 0; mt < 8; ++mt) {
    if (mt % U != w) continue;
    const int d0 = 16 * mt + r0;
    if (kOutBf16) {
      __nv_bfloat16 *o0 = reinterpret_cast<__nv_bfloat16 *>(OUT + c2 * pitch);
      __nv_bfloat16 *o1 = reinterpret_cast<__nv_bfloat16 *>(OUT + (c2 + 1) * pitch);
      if (g0) {
        o0[d0] = __float2bfloat16_rn(o[mt][0]);
        o0[d0 + 8] = __float2bfloat16_rn(o[mt][2]);
      }
      if (g1) {
        o1[d0] = __float2bfloat16_rn(o[mt][1]);
        o1[d0 + 8] = __float2bfloat16_rn(o[mt][3]);
      }
    } else {
      float *o0 = reinterpret_cast<float *>(OUT + c2 * pitch);
      float *o1 = reinterpret_cast<float *>(OUT + (c2 + 1) * pitch);
      if (g0) {
        o0[d0] = o[mt][0];
        o0[d0 + 8] = o[mt][2];
      }
      if (g1) {
        o1[d0] = o[mt][1];
        o1[d0 + 8] = o[mt][3];
      }
    }
  }
  group_bar(bar_id, GT);
  {
    constexpr int cpr = 128 * osz / 16;  // 16-byte chunks per output row
    unsigned char *gout = reinterpret_cast<unsigned char *>(p.out) +
                          x.krow * G * 128 * osz;
    for (int i = gt; i < G * cpr; i += GT) {
      const int g = i / cpr, ch = i % cpr;
      *reinterpret_cast<int4 *>(gout + (size_t)g * 128 * osz + ch * 16) =
          *reinterpret_cast<const int4 *>(OUT + g * pitch + ch * 16);
    }
  }

  // 9. TopB with the window: evict the lowest (score, -position) candidate.
  int victim = -1;
  if (p.evict && n > p.budget + p.window) {
    const int wlo = t - p.window;
    unsigned long long best = ~0ull;
    int bi = -1;
    for (int i = gt; i < n; i += GT) {
      const int pi = i < m ? PS[i] : t;
      if (pi <= wlo) {
        const unsigned long long key =
            ((unsigned long long)__float_as_uint(SC[i]) << 32) |
            (unsigned long long)(0xFFFFFFFFu - (unsigned)pi);
        if (key < best) {
          best = key;
          bi = i;
        }
      }
    }
#pragma unroll
    for (int o2 = 16; o2 > 0; o2 >>= 1) {
      const unsigned long long ob = __shfl_xor_sync(0xffffffffu, best, o2);
      const int oi = __shfl_xor_sync(0xffffffffu, bi, o2);
      if (ob < best) {
        best = ob;
        bi = oi;
      }
    }
    if (U > 1) {
      uint32_t *XW = reinterpret_cast<uint32_t *>(XS);
      if (lane == 0) {
        XW[w * kXsWords + 16] = (uint32_t)best;
        XW[w * kXsWords + 17] = (uint32_t)(best >> 32);
        XW[w * kXsWords + 18] = (uint32_t)bi;
      }
      group_bar(bar_id, GT);
#pragma unroll
      for (int v = 0; v < U; ++v) {
        const unsigned long long kb =
            ((unsigned long long)XW[v * kXsWords + 17] << 32) | XW[v * kXsWords + 16];
        if (kb < best) {
          best = kb;
          bi = (int)XW[v * kXsWords + 18];
        }
      }
    }
    victim = bi;
  }

  // 10. Write back the kept rows' scores, the new row into the freed slot (or
  //     the first free slot when nothing is evicted), length and position.
  float *gsc = p.c.score + x.ug * p.c.sstride;
  int32_t *gps = p.c.pos + x.ug * p.c.sstride;
  const float new_score = SC[m];
  for (int i = gt; i < m; i += GT) gsc[i] = i == victim ? new_score : SC[i];
  const int slot = victim < 0 ? m : (victim < m ? victim : -1);
  if (w == 0) {
    if (slot >= 0) {
      const int chunk = lane & 15;
      __nv_bfloat16 *dst =
          reinterpret_cast<__nv_bfloat16 *>(lane < 16 ? p.c.K : p.c.V) +
          (x.ug * (size_t)p.c.cap + slot) * 128;
      const unsigned char *src = lane < 16 ? KN : VN;
      reinterpret_cast<int4 *>(dst)[chunk] =
          *reinterpret_cast<const int4 *>(src + chunk * 16);
      if (lane == 0) {
        gps[slot] = t;
        if (slot == m) gsc[m] = new_score;
      }
    }
    if (lane == 0) {
      p.c.state[4 * x.ug] = victim < 0 ? m + 1 : m;
      p.c.state[4 * x.ug + 1] = t + 1;
    }
  }
}

template <int T, int U, bool kOutBf16>
__global__ void __launch_bounds__(kMaxThreads, 1)
    fused_step_kernel(const __grid_constant__ CUtensorMap tmK,
                      const __grid_constant__ CUtensorMap tmV,
                      const FusedParams p) {
  extern __shared__ unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kMaxStages];
  __shared__ __align__(8) uint64_t empty_bar[kMaxStages];
  __shared__ int issued_k[kMaxStages];
  __shared__ int consumed_k[kMaxStages];
  __shared__ volatile int s_abort;
  __shared__ volatile int s_ok[kMaxGroups];
  unsigned char *smem = reinterpret_cast<unsigned char *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_units = p.c.S * p.nl * p.c.H;
  const int mine = (int)blockIdx.x < n_units
                       ? (n_units - 1 - (int)blockIdx.x) / (int)gridDim.x + 1
                       : 0;
  const StageLayout L(16 * T);
  const int consumers = p.n_groups * U;

  if (threadIdx.x == 0) {
    for (int s = 0; s < p.n_stages; ++s) {
      mbar_init(smem_u32(&full_bar[s]), 1);
      mbar_init(smem_u32(&empty_bar[s]), 1);
      issued_k[s] = -1;
      consumed_k[s] = -1;
    }
    s_abort = 0;
    fence_mbar_init();
  }
  // Query rows of heads >= G are never copied: zero them once per stage.
  for (int s = 0; s < p.n_stages; ++s) {
    unsigned char *q = smem + s * L.bytes + L.q;
    for (int i = threadIdx.x; i < (8 - p.c.G) * (kQPitch / 16);
         i += blockDim.x)
      reinterpret_cast<int4 *>(q + p.c.G * kQPitch)[i] = make_int4(0, 0, 0, 0);
  }
  fence_proxy_async();
  __syncthreads();

  if (warp == consumers) {
    if (lane == 0) {
      for (int k = 0; k < mine; ++k) {
        const int s = k % p.n_stages;
        const uint32_t ph = (uint32_t)(k / p.n_stages) & 1u;
        if (!mbar_wait(smem_u32(&empty_bar[s]), ph ^ 1u, &s_abort)) {
          atomicOr(p.c.err, ERR_TIMEOUT);
          s_abort = 1;
          break;
        }
        issue_unit(p, &tmK, &tmV, smem + s * L.bytes, smem_u32(&full_bar[s]),
                   (int)blockIdx.x + k * (int)gridDim.x);
        issued_k[s] = k;
      }
    }
  } else if (warp < consumers) {
    const int grp = warp / U, w = warp % U, bar_id = 1 + grp;
    for (int k = grp; k < mine; k += p.n_groups) {
      const int s = k % p.n_stages;
      const uint32_t ph = (uint32_t)(k / p.n_stages) & 1u;
      // One warp waits (bounded) and tells the group, so that every warp
      // of the group takes the same branch before the next named barrier.
      if (w == 0) {
        const bool ok = mbar_wait(smem_u32(&full_bar[s]), ph, &s_abort);
        if (lane == 0) {
          s_ok[grp] = ok ? 1 : 0;
          if (!ok) {
            atomicOr(p.c.err, ERR_TIMEOUT);
            s_abort = 1;
          }
        }
      }
      group_bar(bar_id, 32 * U);
      if (!s_ok[grp]) break;
      mbar_try_wait(smem_u32(&full_bar[s]), ph);  // acquire for this thread
      process_unit<T, U, kOutBf16>(p, smem + s * L.bytes,
                                   (int)blockIdx.x + k * (int)gridDim.x, w,
                                   lane, bar_id);
      fence_proxy_async();
      group_bar(bar_id, 32 * U);
      if (w == 0 && lane == 0) {
        consumed_k[s] = k;
        mbar_arrive(smem_u32(&empty_bar[s]));
      }
    }
  }
  __syncthreads();
  // After an abort, wait (bounded) for copies still landing in our stages.
  if (s_abort && threadIdx.x == 0) {
    volatile int never = 0;
    for (int s = 0; s < p.n_stages; ++s) {
      const int k = issued_k[s];
      if (k >= 0 && consumed_k[s] != k)
        mbar_wait(smem_u32(&full_bar[s]), (uint32_t)(k / p.n_stages) & 1u,
                  &never);
    }
  }
}

template <int T, int U, bool kOutBf16>
cudaError_t launch_tu(const CUtensorMap &tmK, const CUtensorMap &tmV,
                      const FusedParams &p, int grid, int smem_bytes,
                      cudaStream_t st) {
  auto kern = fused_step_kernel<T, U, kOutBf16>;
  cudaError_t e = cudaFuncSetAttribute(
      kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes);
  if (e != cudaSuccess) return e;
  const int threads = 32 * (p.n_groups * U + 1);
  kern<<<grid, threads, smem_bytes, st>>>(tmK, tmV, p);
  return cudaGetLastError();
}

template <bool kOutBf16>
cudaError_t launch_t(const CUtensorMap &tmK, const CUtensorMap &tmV,
                     const FusedParams &p, int grid, int smem_bytes,
                     cudaStream_t st) {
  switch (p.R / 16) {
    case 1: return launch_tu<1, 1, kOutBf16>(tmK, tmV, p, grid, smem_bytes, st);
    case 2: return launch_tu<2, 2, kOutBf16>(tmK, tmV, p, grid, smem_bytes, st);
    case 3: return launch_tu<3, 3, kOutBf16>(tmK, tmV, p, grid, smem_bytes, st);
    case 4: return launch_tu<4, 4, kOutBf16>(tmK, tmV, p, grid, smem_bytes, st);
    case 5: return launch_tu<5, 5, kOutBf16>(tmK, tmV, p, grid, smem_bytes, st);
    case 6: return launch_tu<6, 3, kOutBf16>(tmK, tmV, p, grid, smem_bytes, st);
    case 7: return launch_tu<7, 4, kOutBf16>(tmK, tmV, p, grid, smem_bytes, st);
    case 8: return launch_tu<8, 4, kOutBf16>(tmK, tmV, p, grid, smem_bytes, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace

int fused_stage_bytes(int R) { return (int)StageLayout(R).bytes; }

int fused_group_warps(int R) {
  static const int u[9] = {0, 1, 2, 3, 4, 5, 3, 4, 4};
  return (R % 16 == 0 && R >= 16 && R <= 128) ? u[R / 16] : 0;
}

int fused_max_threads() { return kMaxThreads; }

cudaError_t launch_fused_step(const CUtensorMap &tmK, const CUtensorMap &tmV,
                              const FusedParams &p, int grid, int smem_bytes,
                              cudaStream_t st) {
  if (fused_group_warps(p.R) == 0 || p.n_groups < 1 ||
      p.n_groups > kMaxGroups || p.n_stages > kMaxStages ||
      32 * (p.n_groups * fused_group_warps(p.R) + 1) > kMaxThreads)
    return cudaErrorInvalidValue;
  return p.c.out_bf16 ? launch_t<true>(tmK, tmV, p, grid, smem_bytes, st)
                      : launch_t<false>(tmK, tmV, p, grid, smem_bytes, st);
}

}  // namespace kvr
