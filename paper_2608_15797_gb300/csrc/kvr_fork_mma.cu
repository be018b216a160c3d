// kvr_fork_mma.cu -- the candidate-batched decode step on tensor cores
// (stepwise best-of-N, Sec. 2.2 Eq. 2 and App. C): N candidates share
// the parent's live rows as a read-only prefix; each has a private tail.
// bf16, head_dim 128, G <= 8, N <= 8.
//
// One CTA per (sequence, layer, KV head), one warp per candidate.  The
// prefix K and V rows are copied once (TMA, 16-row boxes, 128B swizzle) into
// shared memory and read by every warp: each prefix row crosses HBM once for
// all N x G query rows.  Each warp then streams its own tail through a
// two-slot TMA ring, inserting its new row, and runs QK^T and PV on bf16
// mma.sync with an online softmax over prefix + tail (P split hi + lo).  The
// scaled logits stay in shared memory, so the candidate's accumulated
// attention (Sec. 2.1, mean over the G heads) is updated with exact
// probabilities after the pass.
#include <cuda.h>
#include <cuda_bf16.h>
#include <math.h>
#include <stdint.h>

#include "kvr_internal.h"
#include "kvr_ptx.cuh"

namespace kvr {
namespace {

using namespace ptx;

constexpr int kBox = 16;                    // rows per TMA box and per tile
constexpr int kTileBytes = 4 * kBox * 128;  // K0, K1, V0, V1 of one tile
constexpr int kQPitch = 272;
constexpr int kMaxCand = 8;

// Shared memory layout (bytes from a 1024-aligned base).
struct ForkMmaLayout {
  int prefix, ring, q, lg, bytes, lg_stride;
  __host__ __device__ ForkMmaLayout(int np_max, int nt_max, int N) {
    const int tp = (np_max + kBox - 1) / kBox;
    prefix = 0;                                   // [tp tiles] K0 K1 V0 V1
    ring = prefix + tp * kTileBytes;              // [N][2 slots] tiles
    q = ring + N * 2 * kTileBytes;                // [N][8][kQPitch]
    lg_stride = ((np_max + nt_max + 1) + 3) & ~3; // logits per head
    lg = q + N * 8 * kQPitch;                     // [N][8][lg_stride] floats
    bytes = lg + N * 8 * lg_stride * 4;
  }
};

__device__ __forceinline__ uint32_t swz(int row, int chunk) {
  return row * 128 + (((chunk & 7) ^ (row & 7)) << 4);
}

// One 16-row tile of the flash pass for one warp (candidate).  K and V point
// at the tile's 128B-swizzled halves; rows >= n_valid are masked; the logits
// of valid rows are stored at LG[g * stride + lg_base + row].
__device__ __forceinline__ void tile_pass(
    const unsigned char *K0, const unsigned char *K1, const unsigned char *V0,
    const unsigned char *V1, int n_valid, const uint32_t (&qb)[8][2],
    float scale_log2e, int G, float *LG, int stride, int lg_base, float &m0,
    float &m1, float &l0, float &l1, float (&o)[8][4], int lane) {
  const int r0l = lane >> 2, c2 = (lane & 3) * 2;
  float s[4] = {0.f, 0.f, 0.f, 0.f}, s2[4] = {0.f, 0.f, 0.f, 0.f};
  {
    const int row = (lane & 7) + ((lane >> 3) & 1) * 8;
#pragma unroll
    for (int ks = 0; ks < 8; ++ks) {
      const int cc = ((ks & 3) << 1) + (lane >> 4);
      const uint32_t addr = smem_u32(ks >> 2 ? K1 : K0) + swz(row, cc);
      uint32_t a0, a1, a2, a3;
      ldsm_x4(addr, a0, a1, a2, a3);
      if (ks & 1) mma_bf16(s2, a0, a1, a2, a3, qb[ks][0], qb[ks][1]);
      else mma_bf16(s, a0, a1, a2, a3, qb[ks][0], qb[ks][1]);
    }
  }
  const int ra = r0l, rb = r0l + 8;
  s[0] = ra < n_valid ? (s[0] + s2[0]) * scale_log2e : -INFINITY;
  s[1] = ra < n_valid ? (s[1] + s2[1]) * scale_log2e : -INFINITY;
  s[2] = rb < n_valid ? (s[2] + s2[2]) * scale_log2e : -INFINITY;
  s[3] = rb < n_valid ? (s[3] + s2[3]) * scale_log2e : -INFINITY;
  if (ra < n_valid) {
    if (c2 < G) LG[c2 * stride + lg_base + ra] = s[0];
    if (c2 + 1 < G) LG[(c2 + 1) * stride + lg_base + ra] = s[1];
  }
  if (rb < n_valid) {
    if (c2 < G) LG[c2 * stride + lg_base + rb] = s[2];
    if (c2 + 1 < G) LG[(c2 + 1) * stride + lg_base + rb] = s[3];
  }
  float x0 = fmaxf(s[0], s[2]), x1 = fmaxf(s[1], s[3]);
#pragma unroll
  for (int off = 4; off < 32; off <<= 1) {
    x0 = fmaxf(x0, __shfl_xor_sync(0xffffffffu, x0, off));
    x1 = fmaxf(x1, __shfl_xor_sync(0xffffffffu, x1, off));
  }
  const float n0 = fmaxf(m0, x0), n1 = fmaxf(m1, x1);  // row 0 is valid
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
  const int row = (lane & 7) + ((lane >> 4) << 3);
#pragma unroll
  for (int mt = 0; mt < 8; ++mt) {
    const int c16 = 2 * mt + ((lane >> 3) & 1);
    const uint32_t addr = smem_u32(c16 >> 3 ? V1 : V0) + swz(row, c16);
    uint32_t v0, v1, v2, v3;
    ldsm_x4_t(addr, v0, v1, v2, v3);
    mma_bf16(o[mt], v0, v1, v2, v3, bp0, bp1);
    mma_bf16(o[mt], v0, v1, v2, v3, bl0, bl1);
  }
}

template <bool kOutBf16>
__global__ void __launch_bounds__(32 * kMaxCand)
    fork_mma_kernel(const __grid_constant__ CUtensorMap tmK,
                    const __grid_constant__ CUtensorMap tmV,
                    const __grid_constant__ CUtensorMap tmTK,
                    const __grid_constant__ CUtensorMap tmTV,
                    const ForkMmaParams p) {
  pdl_begin();
  extern __shared__ unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t pre_bar;
  __shared__ __align__(8) uint64_t ring_bar[kMaxCand][2];
  __shared__ volatile int s_abort;
  unsigned char *smem = reinterpret_cast<unsigned char *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const ForkView &f = p.f;
  const CacheView &c = f.p;
  const int G = c.G, N = f.N;
  const ForkMmaLayout Ly(p.np_max, p.nt_max, N);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int idx = blockIdx.x;
  const int h = idx % c.H, lr = (idx / c.H) % p.nl, sq = idx / (c.H * p.nl);
  const size_t units = (size_t)c.S * c.L * c.H;
  const size_t ug = ((size_t)sq * c.L + p.lb + lr) * c.H + h;
  const int np = c.state[4 * ug], base_pos = c.state[4 * ug + 1];
  const int tp = (np + kBox - 1) / kBox;
  if (np > p.np_max) {  // the host sized shared memory for np_max
    if (threadIdx.x == 0) atomicOr(c.err, ERR_LENGTH);
    return;
  }

  if (threadIdx.x == 0) {
    mbar_init(smem_u32(&pre_bar), 1);
    for (int w = 0; w < N; ++w) {
      mbar_init(smem_u32(&ring_bar[w][0]), 1);
      mbar_init(smem_u32(&ring_bar[w][1]), 1);
    }
    s_abort = 0;
    fence_mbar_init();
  }
  __syncthreads();
  // The prefix: tp boxes of 16 rows per quarter, one transaction.
  if (threadIdx.x == 0 && tp > 0) {
    const uint32_t b = smem_u32(&pre_bar);
    mbar_expect_tx(b, (uint32_t)tp * kTileBytes);
    for (int t = 0; t < tp; ++t) {
      const uint32_t dst = smem_u32(smem + Ly.prefix + t * kTileBytes);
      const int y = (int)(ug * (size_t)c.cap) + t * kBox;
      tma_load_2d(dst, &tmK, 0, y, b);
      tma_load_2d(dst + kBox * 128, &tmK, 64, y, b);
      tma_load_2d(dst + 2 * kBox * 128, &tmV, 0, y, b);
      tma_load_2d(dst + 3 * kBox * 128, &tmV, 64, y, b);
    }
  }

  const int cand = warp;
  const size_t cu = (size_t)cand * units + ug;
  const int nt0 = cand < N ? f.tlen[cu] : 0;  // tail rows before the append
  if (cand < N && lane == 0 && (nt0 + 1 > f.tcap || nt0 > p.nt_max))
    atomicOr(c.err, ERR_CAPACITY);
  const bool active = cand < N && nt0 + 1 <= f.tcap && nt0 <= p.nt_max;
  const int ntot = nt0 + 1;                   // with the new row
  const int tt = (ntot + kBox - 1) / kBox;    // tail tiles
  const size_t kv_row = (((size_t)cand * c.S + sq) * p.nl + lr) * c.H + h;
  unsigned char *ring = smem + Ly.ring + warp * 2 * kTileBytes;
  auto issue_tail = [&](int k) {  // tail tile k into slot k & 1 (lane 0)
    const uint32_t b = smem_u32(&ring_bar[warp][k & 1]);
    const int live = min(kBox, nt0 - k * kBox);  // slab rows of this tile
    if (live <= 0) {
      mbar_arrive(b);  // nothing to copy: only the new row, from the inputs
      return;
    }
    mbar_expect_tx(b, kTileBytes);
    const uint32_t dst = smem_u32(ring + (k & 1) * kTileBytes);
    const int y = (int)(cu * (size_t)f.tcap) + k * kBox;
    tma_load_2d(dst, &tmTK, 0, y, b);
    tma_load_2d(dst + kBox * 128, &tmTK, 64, y, b);
    tma_load_2d(dst + 2 * kBox * 128, &tmTV, 0, y, b);
    tma_load_2d(dst + 3 * kBox * 128, &tmTV, 64, y, b);
  };
  if (active && lane == 0) {
    issue_tail(0);
    if (tt > 1) issue_tail(1);
  }
  // Query rows of this candidate (zero beyond G).
  unsigned char *Q = smem + Ly.q + warp * 8 * kQPitch;
  if (active) {
    const int4 *qg = reinterpret_cast<const int4 *>(p.q + kv_row * G * 128);
    for (int i = lane; i < 8 * 16; i += 32) {
      const int g = i >> 4, ch = i & 15;
      *reinterpret_cast<int4 *>(Q + g * kQPitch + ch * 16) =
          g < G ? qg[g * 16 + ch] : make_int4(0, 0, 0, 0);
    }
  }
  // The prefix is shared: wait for it, zero V beyond np once, then barrier.
  if (tp > 0 && !mbar_wait(smem_u32(&pre_bar), 0u, &s_abort)) {
    if (threadIdx.x == 0) atomicOr(c.err, ERR_TIMEOUT);
    s_abort = 1;
  }
  for (int i = threadIdx.x; i < (tp * kBox - np) * 16; i += blockDim.x) {
    const int r = np + (i >> 4), c16 = i & 15, t = r / kBox, rr = r % kBox;
    *reinterpret_cast<int4 *>(smem + Ly.prefix + t * kTileBytes +
                              (2 + (c16 >> 3)) * kBox * 128 + rr * 128 +
                              (c16 & 7) * 16) = make_int4(0, 0, 0, 0);
  }
  __syncthreads();
  if (!active || s_abort) {
    // Inactive warps only drain nothing; an abort drains the ring below.
  } else {
    uint32_t qb[8][2];
    {
      const uint32_t qa = smem_u32(Q) + (lane & 7) * kQPitch + (lane >> 3) * 16;
#pragma unroll
      for (int i = 0; i < 4; ++i)
        ldsm_x4(qa + i * 64, qb[2 * i][0], qb[2 * i][1], qb[2 * i + 1][0],
                qb[2 * i + 1][1]);
    }
    float *LG = reinterpret_cast<float *>(smem + Ly.lg) + warp * 8 * Ly.lg_stride;
    float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
    float o[8][4];
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
    // Prefix tiles (shared, already in shared memory).
    for (int t = 0; t < tp; ++t) {
      const unsigned char *T0 = smem + Ly.prefix + t * kTileBytes;
      tile_pass(T0, T0 + kBox * 128, T0 + 2 * kBox * 128, T0 + 3 * kBox * 128,
                min(kBox, np - t * kBox), qb, p.scale_log2e, G, LG, Ly.lg_stride,
                t * kBox, m0, m1, l0, l1, o, lane);
    }
    // Tail tiles (private, streamed).
    for (int k = 0; k < tt; ++k) {
      if (!mbar_wait(smem_u32(&ring_bar[warp][k & 1]), (uint32_t)(k >> 1) & 1u,
                     &s_abort)) {
        if (lane == 0) {
          atomicOr(c.err, ERR_TIMEOUT);
          s_abort = 1;
        }
        break;
      }
      unsigned char *T0 = ring + (k & 1) * kTileBytes;
      unsigned char *K0 = T0, *K1 = T0 + kBox * 128;
      unsigned char *V0 = T0 + 2 * kBox * 128, *V1 = T0 + 3 * kBox * 128;
      const int valid = min(kBox, ntot - k * kBox);
      const int rn = nt0 - k * kBox;  // the new row, if in this tile
      if (rn >= 0 && rn < kBox) {
        const int ch = lane & 15;
        unsigned char *dst = lane < 16 ? (ch < 8 ? K0 : K1) : (ch < 8 ? V0 : V1);
        const __nv_bfloat16 *src = (lane < 16 ? p.k_new : p.v_new) + kv_row * 128;
        *reinterpret_cast<int4 *>(dst + swz(rn, ch)) =
            reinterpret_cast<const int4 *>(src)[ch];
      }
      for (int i = lane; i < (kBox - valid) * 16; i += 32) {
        const int r = valid + (i >> 4), c16 = i & 15;
        *reinterpret_cast<int4 *>((c16 < 8 ? V0 : V1) + r * 128 + (c16 & 7) * 16) =
            make_int4(0, 0, 0, 0);
      }
      __syncwarp();
      tile_pass(K0, K1, V0, V1, valid, qb, p.scale_log2e, G, LG, Ly.lg_stride,
                np + k * kBox, m0, m1, l0, l1, o, lane);
      fence_proxy_async();
      __syncwarp();
      if (lane == 0 && k + 2 < tt) issue_tail(k + 2);
    }
    if (!s_abort) {
#pragma unroll
      for (int off = 4; off < 32; off <<= 1) {
        l0 += __shfl_xor_sync(0xffffffffu, l0, off);
        l1 += __shfl_xor_sync(0xffffffffu, l1, off);
      }
      const float i0 = 1.f / l0, i1 = 1.f / l1;
      if (lane < 4 && !(l0 >= 1.f && l0 < INFINITY && l1 >= 1.f && l1 < INFINITY))
        atomicOr(c.err, ERR_NONFINITE);
      // Output of this candidate (fragments -> rows via movmatrix for bf16).
      const int c2 = (lane & 3) * 2, r0l = lane >> 2;
      constexpr int osz = kOutBf16 ? 2 : 4;
      unsigned char *gout = reinterpret_cast<unsigned char *>(p.out) +
                            kv_row * G * 128 * osz;
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) {
        if (kOutBf16) {
          const uint32_t lo = movm_t(pack_bf16(o[mt][0] * i0, o[mt][1] * i1));
          const uint32_t hi = movm_t(pack_bf16(o[mt][2] * i0, o[mt][3] * i1));
          const int g = lane >> 2, dd = 16 * mt + 2 * (lane & 3);
          if (g < G) {
            *reinterpret_cast<uint32_t *>(gout + ((size_t)g * 128 + dd) * 2) = lo;
            *reinterpret_cast<uint32_t *>(gout + ((size_t)g * 128 + dd + 8) * 2) = hi;
          }
        } else {
          float *of = reinterpret_cast<float *>(gout);
          const int d0 = 16 * mt + r0l;
          if (c2 < G) {
            of[c2 * 128 + d0] = o[mt][0] * i0;
            of[c2 * 128 + d0 + 8] = o[mt][2] * i0;
          }
          if (c2 + 1 < G) {
            of[(c2 + 1) * 128 + d0] = o[mt][1] * i1;
            of[(c2 + 1) * 128 + d0 + 8] = o[mt][3] * i1;
          }
        }
      }
      // Per-head max and 1/sum for the exact probabilities: lanes 0..3 hold
      // columns c2, c2 + 1; broadcast by shuffles.
      float Mg[8], iLg[8];
#pragma unroll
      for (int g = 0; g < 8; ++g) {
        const int src = g >> 1;
        const float mm = __shfl_sync(0xffffffffu, (g & 1) ? m1 : m0, src);
        const float ii = __shfl_sync(0xffffffffu, (g & 1) ? i1 : i0, src);
        Mg[g] = mm;
        iLg[g] = ii;
      }
      __syncwarp();
      // Accumulated attention of the candidate: prefix copy and tail.
      float *ps = f.pscore + cu * (size_t)c.sstride;
      float *ts = f.tscore + cu * (size_t)f.tstride;
      const float inv_g = 1.f / (float)G;
      for (int i = lane; i < np + ntot; i += 32) {
        float acc = 0.f;
#pragma unroll
        for (int g = 0; g < 8; ++g)
          if (g < G) acc += exp2f(LG[g * Ly.lg_stride + i] - Mg[g]) * iLg[g];
        acc *= inv_g;
        if (i < np) ps[i] += acc;
        else if (i - np < nt0) ts[i - np] += acc;
        else ts[nt0] = acc;
      }
      // Append the new row to the tail.
      if (lane < 16) {
        __nv_bfloat16 *dk = reinterpret_cast<__nv_bfloat16 *>(f.TK) +
                            (cu * (size_t)f.tcap + nt0) * 128;
        reinterpret_cast<int4 *>(dk)[lane] =
            reinterpret_cast<const int4 *>(p.k_new + kv_row * 128)[lane];
      } else {
        __nv_bfloat16 *dv = reinterpret_cast<__nv_bfloat16 *>(f.TV) +
                            (cu * (size_t)f.tcap + nt0) * 128;
        reinterpret_cast<int4 *>(dv)[lane - 16] =
            reinterpret_cast<const int4 *>(p.v_new + kv_row * 128)[lane - 16];
      }
      if (lane == 0) {
        f.tpos[cu * f.tstride + nt0] = base_pos + nt0;
        f.tlen[cu] = ntot;
      }
    }
  }
  __syncthreads();
  if (s_abort && active && lane == 0) {  // drain this warp's ring (bounded)
    volatile int never = 0;
    for (int k = max(0, tt - 2); k < tt; ++k)
      mbar_wait(smem_u32(&ring_bar[warp][k & 1]), (uint32_t)(k >> 1) & 1u, &never);
  }
}

}  // namespace

size_t fork_mma_smem_bytes(int np_max, int nt_max, int n_cand) {
  return (size_t)ForkMmaLayout(np_max, nt_max, n_cand).bytes + 1024;
}
int fork_mma_box_rows() { return kBox; }
int fork_mma_max_cand() { return kMaxCand; }

cudaError_t launch_fork_mma(const CUtensorMap &tmK, const CUtensorMap &tmV,
                            const CUtensorMap &tmTK, const CUtensorMap &tmTV,
                            const ForkMmaParams &p, cudaStream_t st) {
  const int smem = (int)fork_mma_smem_bytes(p.np_max, p.nt_max, p.f.N);
  const int units = p.f.p.S * p.nl * p.f.p.H;
  const int threads = 32 * p.f.N;
  cudaError_t e;
  if (p.f.p.out_bf16) {
    e = cudaFuncSetAttribute(fork_mma_kernel<true>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(fork_mma_kernel<true>, dim3(units), dim3(threads), smem,
                      st, tmK, tmV, tmTK, tmTV, p);
  } else {
    e = cudaFuncSetAttribute(fork_mma_kernel<false>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(fork_mma_kernel<false>, dim3(units), dim3(threads), smem,
                      st, tmK, tmV, tmTK, tmTV, p);
  }
}

}  // namespace kvr
