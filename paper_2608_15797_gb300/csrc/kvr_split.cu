// kvr_split.cu -- full-context decode attention split over the rows (the
// KV-Rescue helper keeps its full cache, Sec. 3.1 / App. D): append the new
// row and compute Attn(q_t, C) (Eq. 1) over every cached row, with no
// importance scores and no eviction.  bf16, head_dim 128, G <= 8.
//
// split_partial_kernel: grid (splits, units).  Each CTA takes a contiguous
//   chunk of a unit's rows and streams it through shared memory in 64-row
//   stages (two 128B-swizzled TMA boxes for K and two for V per stage,
//   double-buffered on mbarriers).  Each of the 4 warps owns one 16-row tile
//   per stage: QK^T and PV on bf16 mma.sync (P split hi + lo), with an online
//   softmax (running max and sum per query head).  The warps' states are
//   merged in shared memory and the CTA writes its (max, sum, unnormalised
//   output) to the workspace.
// split_combine_kernel: grid (units).  Merges the splits of a unit into the
//   output, then appends the new row to the cache (the partial kernels only
//   read the slab, so nothing races).
#include <cuda.h>
#include <cuda_bf16.h>
#include <math.h>
#include <stdint.h>

#include "kvr_internal.h"
#include "kvr_ptx.cuh"

namespace kvr {
namespace {

using namespace ptx;

constexpr int kRows = 64;                     // rows per stage
constexpr int kWarps = 4;                     // one 16-row tile each
constexpr int kStages = 2;
constexpr int kBox = kRows * 128;             // bytes of one 64-column box
constexpr int kStageBytes = 4 * kBox;         // K0, K1, V0, V1
constexpr int kQPitch = 272;
constexpr int kWsStride = 130;                // floats per (split, head)

struct SmemLayout {
  static constexpr int q = kStages * kStageBytes;
  static constexpr int ml = q + 8 * kQPitch;  // [warp][8] max, [warp][8] sum
  static constexpr int bytes = ml + 2 * kWarps * 8 * 4;
};

__global__ void __launch_bounds__(32 * kWarps)
    split_partial_kernel(const __grid_constant__ CUtensorMap tmK,
                         const __grid_constant__ CUtensorMap tmV,
                         const SplitParams p) {
  pdl_begin();
  extern __shared__ unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kStages];
  __shared__ volatile int s_abort;
  unsigned char *smem = reinterpret_cast<unsigned char *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const CacheView &c = p.c;
  const int G = c.G;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int split = blockIdx.x, idx = blockIdx.y;
  const int h = idx % c.H, lr = (idx / c.H) % p.nl, sq = idx / (c.H * p.nl);
  const size_t ug = ((size_t)sq * c.L + p.lb + lr) * c.H + h;
  const size_t krow = ((size_t)sq * p.nl + lr) * c.H + h;
  const int len = c.state[4 * ug];
  const int n = len + 1;
  int chunk = (n + p.n_splits - 1) / p.n_splits;
  chunk = (chunk + kRows - 1) / kRows * kRows;
  const int r0 = split * chunk, r1 = min(n, r0 + chunk);
  float *ws = p.ws + (((size_t)idx * p.n_splits + split) * G) * kWsStride;
  if (r0 >= r1) {  // an empty split contributes nothing
    for (int g = threadIdx.x; g < G; g += blockDim.x) {
      ws[g * kWsStride] = -INFINITY;
      ws[g * kWsStride + 1] = 0.f;
    }
    return;
  }
  const int n_st = (r1 - r0 + kRows - 1) / kRows;
  const int row0 = (int)(ug * (size_t)c.cap) + r0;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) mbar_init(smem_u32(&full_bar[s]), 1);
    s_abort = 0;
    fence_mbar_init();
  }
  // Query rows (zero beyond G) with plain loads; bounded by 8 x 256 bytes.
  {
    const int4 *qg = reinterpret_cast<const int4 *>(p.q + krow * G * 128);
    for (int i = threadIdx.x; i < 8 * 16; i += blockDim.x) {
      const int g = i >> 4, ch = i & 15;
      *reinterpret_cast<int4 *>(smem + SmemLayout::q + g * kQPitch + ch * 16) =
          g < G ? qg[g * 16 + ch] : make_int4(0, 0, 0, 0);
    }
  }
  __syncthreads();
  auto issue = [&](int st) {
    const uint32_t b = smem_u32(&full_bar[st % kStages]);
    const uint32_t dst = smem_u32(smem + (st % kStages) * kStageBytes);
    mbar_expect_tx(b, kStageBytes);
    const int y = row0 + st * kRows;
    tma_load_2d(dst, &tmK, 0, y, b);
    tma_load_2d(dst + kBox, &tmK, 64, y, b);
    tma_load_2d(dst + 2 * kBox, &tmV, 0, y, b);
    tma_load_2d(dst + 3 * kBox, &tmV, 64, y, b);
  };
  if (threadIdx.x == 0)
    for (int st = 0; st < min(kStages, n_st); ++st) issue(st);

  uint32_t qb[8][2];
  {
    const uint32_t qa = smem_u32(smem + SmemLayout::q) + (lane & 7) * kQPitch +
                        (lane >> 3) * 16;
#pragma unroll
    for (int i = 0; i < 4; ++i)
      ldsm_x4(qa + i * 64, qb[2 * i][0], qb[2 * i][1], qb[2 * i + 1][0],
              qb[2 * i + 1][1]);
  }
  const int r0l = lane >> 2, c2 = (lane & 3) * 2;
  float m0 = -INFINITY, m1 = -INFINITY;  // running max of columns c2, c2+1
  float l0 = 0.f, l1 = 0.f;              // this lane's share of the sums
  float o[8][4];
#pragma unroll
  for (int mt = 0; mt < 8; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;

  for (int st = 0; st < n_st; ++st) {
    const int buf = st % kStages;
    if (!mbar_wait(smem_u32(&full_bar[buf]), (uint32_t)(st / kStages) & 1u,
                   &s_abort)) {
      if (lane == 0) {
        atomicOr(c.err, ERR_TIMEOUT);
        s_abort = 1;
      }
      break;
    }
    unsigned char *K0 = smem + buf * kStageBytes, *K1 = K0 + kBox;
    unsigned char *V0 = K0 + 2 * kBox, *V1 = K0 + 3 * kBox;
    const int base = r0 + st * kRows;  // unit row of stage row 0
    const int t0 = warp * 16;          // this warp's tile in the stage
    // The new row (unit row len) comes from the inputs; rows at or beyond
    // the chunk end are masked and their V zeroed (they may hold anything).
    {
      const int rn = len - base;
      if (rn >= t0 && rn < t0 + 16) {
        const int chunk16 = lane & 15, half = chunk16 >> 3, cc = chunk16 & 7;
        const uint32_t off = rn * 128 + ((cc ^ (rn & 7)) << 4);
        unsigned char *dst = lane < 16 ? (half ? K1 : K0) : (half ? V1 : V0);
        const __nv_bfloat16 *src = (lane < 16 ? p.k_new : p.v_new) + krow * 128;
        *reinterpret_cast<int4 *>(dst + off) =
            reinterpret_cast<const int4 *>(src)[chunk16];
      }
      const int lo = max(t0, r1 - base);
      for (int i = lane; i < (t0 + 16 - lo) * 16; i += 32) {
        const int r = lo + (i >> 4), c16 = i & 15;
        if (r >= t0)
          *reinterpret_cast<int4 *>((c16 < 8 ? V0 : V1) + r * 128 +
                                    (c16 & 7) * 16) = make_int4(0, 0, 0, 0);
      }
    }
    __syncwarp();
    if (base + t0 < r1) {
      float s[4] = {0.f, 0.f, 0.f, 0.f}, s2[4] = {0.f, 0.f, 0.f, 0.f};
      {
        const int row = t0 + (lane & 7) + ((lane >> 3) & 1) * 8;
        const uint32_t b0 = smem_u32(K0) + row * 128, b1 = smem_u32(K1) + row * 128;
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
          const int cc = ((ks & 3) << 1) + (lane >> 4);
          const uint32_t addr = (ks >> 2 ? b1 : b0) + ((cc ^ (row & 7)) << 4);
          uint32_t a0, a1, a2, a3;
          ldsm_x4(addr, a0, a1, a2, a3);
          if (ks & 1) mma_bf16(s2, a0, a1, a2, a3, qb[ks][0], qb[ks][1]);
          else mma_bf16(s, a0, a1, a2, a3, qb[ks][0], qb[ks][1]);
        }
      }
      const int ra = base + t0 + r0l, rb = ra + 8;
      s[0] = ra < r1 ? (s[0] + s2[0]) * p.scale_log2e : -INFINITY;
      s[1] = ra < r1 ? (s[1] + s2[1]) * p.scale_log2e : -INFINITY;
      s[2] = rb < r1 ? (s[2] + s2[2]) * p.scale_log2e : -INFINITY;
      s[3] = rb < r1 ? (s[3] + s2[3]) * p.scale_log2e : -INFINITY;
      float x0 = fmaxf(s[0], s[2]), x1 = fmaxf(s[1], s[3]);
#pragma unroll
      for (int off = 4; off < 32; off <<= 1) {
        x0 = fmaxf(x0, __shfl_xor_sync(0xffffffffu, x0, off));
        x1 = fmaxf(x1, __shfl_xor_sync(0xffffffffu, x1, off));
      }
      const float n0 = fmaxf(m0, x0), n1 = fmaxf(m1, x1);  // finite: row ra valid
      const float a0 = exp2f(m0 - n0), a1 = exp2f(m1 - n1);
      m0 = n0;
      m1 = n1;
      s[0] = exp2f(s[0] - m0);
      s[1] = exp2f(s[1] - m1);
      s[2] = exp2f(s[2] - m0);
      s[3] = exp2f(s[3] - m1);
      l0 = l0 * a0 + s[0] + s[2];
      l1 = l1 * a1 + s[1] + s[3];
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) {
        o[mt][0] *= a0;
        o[mt][2] *= a0;
        o[mt][1] *= a1;
        o[mt][3] *= a1;
      }
      const uint32_t h0 = pack_bf16(s[0], s[1]), h1 = pack_bf16(s[2], s[3]);
      const __nv_bfloat162 hb0 = *reinterpret_cast<const __nv_bfloat162 *>(&h0);
      const __nv_bfloat162 hb1 = *reinterpret_cast<const __nv_bfloat162 *>(&h1);
      const uint32_t bp0 = movm_t(h0), bp1 = movm_t(h1);
      const uint32_t bl0 = movm_t(pack_bf16(s[0] - __low2float(hb0), s[1] - __high2float(hb0)));
      const uint32_t bl1 = movm_t(pack_bf16(s[2] - __low2float(hb1), s[3] - __high2float(hb1)));
      const int row = t0 + (lane & 7) + ((lane >> 4) << 3);
      const uint32_t b0 = smem_u32(V0) + row * 128, b1 = smem_u32(V1) + row * 128;
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) {
        const int c16 = 2 * mt + ((lane >> 3) & 1);
        const uint32_t addr = (c16 >> 3 ? b1 : b0) + (((c16 & 7) ^ (row & 7)) << 4);
        uint32_t v0, v1, v2, v3;
        ldsm_x4_t(addr, v0, v1, v2, v3);
        mma_bf16(o[mt], v0, v1, v2, v3, bp0, bp1);
        mma_bf16(o[mt], v0, v1, v2, v3, bl0, bl1);
      }
    }
    // Refill this buffer once every warp is done with it.
    fence_proxy_async();
    __syncthreads();
    if (threadIdx.x == 0 && st + kStages < n_st) issue(st + kStages);
  }
  __syncthreads();
  if (s_abort) {  // drain copies still landing in our buffers (bounded)
    if (threadIdx.x == 0) {
      volatile int never = 0;
      for (int st = 0; st < n_st; ++st)
        mbar_wait(smem_u32(&full_bar[st % kStages]), (uint32_t)(st / kStages) & 1u,
                  &never);
    }
    return;
  }

  // Merge the four warps: common max per head, rescaled sums and outputs.
#pragma unroll
  for (int off = 4; off < 32; off <<= 1) {
    l0 += __shfl_xor_sync(0xffffffffu, l0, off);
    l1 += __shfl_xor_sync(0xffffffffu, l1, off);
  }
  float *ML = reinterpret_cast<float *>(smem + SmemLayout::ml);
  if (lane < 4) {
    ML[warp * 8 + c2] = m0;
    ML[warp * 8 + c2 + 1] = m1;
  }
  __syncthreads();
  float M0 = -INFINITY, M1 = -INFINITY;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) {
    M0 = fmaxf(M0, ML[w * 8 + c2]);
    M1 = fmaxf(M1, ML[w * 8 + c2 + 1]);
  }
  const float f0 = m0 == -INFINITY ? 0.f : exp2f(m0 - M0);
  const float f1 = m1 == -INFINITY ? 0.f : exp2f(m1 - M1);
  float *XO = reinterpret_cast<float *>(smem);  // [warp][mt][4][32]
#pragma unroll
  for (int mt = 0; mt < 8; ++mt) {
    XO[((warp * 8 + mt) * 4 + 0) * 32 + lane] = o[mt][0] * f0;
    XO[((warp * 8 + mt) * 4 + 1) * 32 + lane] = o[mt][1] * f1;
    XO[((warp * 8 + mt) * 4 + 2) * 32 + lane] = o[mt][2] * f0;
    XO[((warp * 8 + mt) * 4 + 3) * 32 + lane] = o[mt][3] * f1;
  }
  if (lane < 4) {
    ML[32 + warp * 8 + c2] = l0 * f0;
    ML[32 + warp * 8 + c2 + 1] = l1 * f1;
  }
  __syncthreads();
  if (warp == 0) {
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        float sum = 0.f;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) sum += XO[((w * 8 + mt) * 4 + e) * 32 + lane];
        const int g = c2 + (e & 1), d = 16 * mt + r0l + 8 * (e >> 1);
        if (g < G) ws[g * kWsStride + 2 + d] = sum;
      }
    }
    if (lane < 4) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int g = c2 + e;
        if (g < G) {
          float L = 0.f;
#pragma unroll
          for (int w = 0; w < kWarps; ++w) L += ML[32 + w * 8 + g];
          ws[g * kWsStride] = e ? M1 : M0;
          ws[g * kWsStride + 1] = L;
        }
      }
    }
  }
}

template <typename O>
__global__ void __launch_bounds__(128) split_combine_kernel(const SplitParams p,
                                                            void *out) {
  pdl_begin();
  const CacheView &c = p.c;
  const int G = c.G, idx = blockIdx.x;
  const int h = idx % c.H, lr = (idx / c.H) % p.nl, sq = idx / (c.H * p.nl);
  const size_t ug = ((size_t)sq * c.L + p.lb + lr) * c.H + h;
  const size_t krow = ((size_t)sq * p.nl + lr) * c.H + h;
  const float *ws = p.ws + (size_t)idx * p.n_splits * G * kWsStride;
  const int d = threadIdx.x;  // 128 threads, one head-dim column each
  O *og = reinterpret_cast<O *>(out) + krow * G * 128;
  for (int g = 0; g < G; ++g) {
    float M = -INFINITY;
    for (int s = 0; s < p.n_splits; ++s) M = fmaxf(M, ws[(s * G + g) * kWsStride]);
    float L = 0.f, acc = 0.f;
    for (int s = 0; s < p.n_splits; ++s) {
      const float *w = ws + (s * G + g) * kWsStride;
      if (w[0] == -INFINITY) continue;  // empty split: its outputs are unset
      const float f = exp2f(w[0] - M);
      L += w[1] * f;
      acc += w[2 + d] * f;
    }
    if (d == 0 && !(L >= 1.f && L < INFINITY)) atomicOr(c.err, ERR_NONFINITE);
    const float v = acc / L;
    if constexpr (sizeof(O) == 2) og[g * 128 + d] = __float2bfloat16_rn(v);
    else og[g * 128 + d] = v;
  }
  // Append the new row now that every split has read the slab.
  const int len = c.state[4 * ug], t = c.state[4 * ug + 1];
  __nv_bfloat16 *K = reinterpret_cast<__nv_bfloat16 *>(c.K) + (ug * c.cap + len) * 128;
  __nv_bfloat16 *V = reinterpret_cast<__nv_bfloat16 *>(c.V) + (ug * c.cap + len) * 128;
  K[d] = p.k_new[krow * 128 + d];
  V[d] = p.v_new[krow * 128 + d];
  __syncthreads();  // every thread has read the state before it changes
  if (d == 0) {
    c.pos[ug * c.sstride + len] = t;
    c.score[ug * c.sstride + len] = 0.f;
    c.state[4 * ug] = len + 1;
    c.state[4 * ug + 1] = t + 1;
    c.state[4 * ug + 2] = 0;  // the R-KV key sum no longer matches
  }
}

}  // namespace

size_t split_workspace_bytes(const CacheView &c, int nl, int n_splits) {
  return (size_t)c.S * nl * c.H * n_splits * c.G * kWsStride * sizeof(float);
}

int split_rows_per_stage() { return kRows; }

cudaError_t launch_split_attend(const CUtensorMap &tmK, const CUtensorMap &tmV,
                                const SplitParams &p, void *out,
                                cudaStream_t st) {
  const int smem = SmemLayout::bytes + 1024;
  cudaError_t e = cudaFuncSetAttribute(
      split_partial_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  const int units = p.c.S * p.nl * p.c.H;
  e = launch_pdl(split_partial_kernel, dim3(p.n_splits, units),
                 dim3(32 * kWarps), smem, st, tmK, tmV, p);
  if (e != cudaSuccess) return e;
  if (p.c.out_bf16)
    return launch_pdl(split_combine_kernel<__nv_bfloat16>, dim3(units),
                      dim3(128), 0, st, p, out);
  return launch_pdl(split_combine_kernel<float>, dim3(units), dim3(128), 0, st,
                    p, out);
}

}  // namespace kvr
