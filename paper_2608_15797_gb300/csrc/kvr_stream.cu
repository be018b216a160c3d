// kvr_stream.cu -- the fused decode step for units too long for the staged
// kernel of kvr_fused.cu (more than its 160 live rows, up to kMaxRows): append +
// Attn(q_t, C) (Eq. 1) + accumulated-attention update (Sec. 2.1) + eviction
// of the single surplus row (TopB of Eq. 1 with the Sec. 4.1 window) +
// in-place compaction, one CTA per (sequence, layer, KV head), K and V each
// read once.  bf16, head_dim 128, G <= 8.
//
// The unit's rows stream through a double-buffered ring of 64-row stages
// filled by TMA in 16-row boxes (so the last stage reads only live rows);
// each of the 4 warps owns one 16-row tile per stage and runs QK^T and PV on
// bf16 mma.sync with an online softmax (P split hi + lo).  The scaled logits
// stay in shared memory, so once the warps' softmax states are merged every
// row's exact probability is available for the score update without a
// second pass over K.
#include <cuda.h>
#include <cuda_bf16.h>
#include <math.h>
#include <stdint.h>

#include "kvr_internal.h"
#include "kvr_ptx.cuh"

namespace kvr {
namespace {

using namespace ptx;

constexpr int kRows = 64;              // rows per stage
constexpr int kBoxRows = 16;           // rows per TMA box
constexpr int kWarps = 4;              // one 16-row tile each per stage
constexpr int kStages = 2;
constexpr int kStageBytes = 4 * kRows * 128;  // K0, K1, V0, V1
constexpr int kQPitch = 272;
constexpr int kMaxRowsStream = 2048;

// Dynamic shared memory layout (bytes from a 1024-aligned base).
struct StreamLayout {
  int q, lg, sc, ps, ns, ml, red, bytes;
  __host__ __device__ explicit StreamLayout(int n_max) {
    const int nm = (n_max + 15) & ~15;
    q = kStages * kStageBytes;
    lg = q + 8 * kQPitch;   // [8][nm] scaled logits
    sc = lg + 8 * nm * 4;   // [nm] old scores
    ps = sc + nm * 4;       // [nm] positions
    ns = ps + nm * 4;       // [nm] new scores
    ml = ns + nm * 4;       // [warp][8] max, [warp][8] sum, [8] M, [8] 1/L
    red = ml + (2 * kWarps + 2) * 8 * 4;  // argmin per warp (key, row)
    bytes = red + kWarps * 16;
  }
};

template <bool kOutBf16>
__global__ void __launch_bounds__(32 * kWarps)
    stream_step_kernel(const __grid_constant__ CUtensorMap tmK,
                       const __grid_constant__ CUtensorMap tmV,
                       const StreamParams p) {
  pdl_begin();
  extern __shared__ unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kStages];
  __shared__ volatile int s_abort;
  unsigned char *smem = reinterpret_cast<unsigned char *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const StreamLayout Ly(p.n_max);
  const int nm = (p.n_max + 15) & ~15;
  const CacheView &c = p.c;
  const int G = c.G;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int idx = blockIdx.x;
  const int h = idx % c.H, lr = (idx / c.H) % p.nl, sq = idx / (c.H * p.nl);
  const size_t ug = ((size_t)sq * c.L + p.lb + lr) * c.H + h;
  const size_t krow = ((size_t)sq * p.nl + lr) * c.H + h;
  const int m = c.state[4 * ug], t = c.state[4 * ug + 1];
  const int n = m + 1;
  if (m < 0 || n > p.n_max) {  // the host sized shared memory for n_max
    if (tid == 0) atomicOr(c.err, ERR_LENGTH);
    return;
  }
  const int n_st = (n + kRows - 1) / kRows;
  const int row0 = (int)(ug * (size_t)c.cap);
  float *LG = reinterpret_cast<float *>(smem + Ly.lg);
  float *SC = reinterpret_cast<float *>(smem + Ly.sc);
  int32_t *PS = reinterpret_cast<int32_t *>(smem + Ly.ps);
  float *NS = reinterpret_cast<float *>(smem + Ly.ns);
  float *ML = reinterpret_cast<float *>(smem + Ly.ml);

  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) mbar_init(smem_u32(&full_bar[s]), 1);
    s_abort = 0;
    fence_mbar_init();
  }
  {
    const int4 *qg = reinterpret_cast<const int4 *>(p.q + krow * G * 128);
    for (int i = tid; i < 8 * 16; i += blockDim.x) {
      const int g = i >> 4, ch = i & 15;
      *reinterpret_cast<int4 *>(smem + Ly.q + g * kQPitch + ch * 16) =
          g < G ? qg[g * 16 + ch] : make_int4(0, 0, 0, 0);
    }
    const float *gsc = c.score + ug * c.sstride;
    const int32_t *gps = c.pos + ug * c.sstride;
    for (int i = tid; i < m; i += blockDim.x) {
      SC[i] = gsc[i];
      PS[i] = gps[i];
    }
  }
  __syncthreads();
  // Stage st holds unit rows [64 st, 64 st + 64); only slab rows < m are
  // copied (16-row boxes), the new row m comes from the inputs.
  auto issue = [&](int st) {
    const uint32_t b = smem_u32(&full_bar[st % kStages]);
    const uint32_t dst = smem_u32(smem + (st % kStages) * kStageBytes);
    const int first = st * kRows;
    const int live = max(0, min(kRows, m - first));
    const int boxes = (live + kBoxRows - 1) / kBoxRows;
    mbar_expect_tx(b, (uint32_t)boxes * 4u * kBoxRows * 128u);
    for (int bx = 0; bx < boxes; ++bx) {
      const int y = row0 + first + bx * kBoxRows;
      const uint32_t off = bx * kBoxRows * 128;
      tma_load_2d(dst + off, &tmK, 0, y, b);
      tma_load_2d(dst + kRows * 128 + off, &tmK, 64, y, b);
      tma_load_2d(dst + 2 * kRows * 128 + off, &tmV, 0, y, b);
      tma_load_2d(dst + 3 * kRows * 128 + off, &tmV, 64, y, b);
    }
  };
  if (tid == 0)
    for (int st = 0; st < min(kStages, n_st); ++st) issue(st);

  uint32_t qb[8][2];
  {
    const uint32_t qa = smem_u32(smem + Ly.q) + (lane & 7) * kQPitch + (lane >> 3) * 16;
#pragma unroll
    for (int i = 0; i < 4; ++i)
      ldsm_x4(qa + i * 64, qb[2 * i][0], qb[2 * i][1], qb[2 * i + 1][0],
              qb[2 * i + 1][1]);
  }
  const int r0l = lane >> 2, c2 = (lane & 3) * 2;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  float o[8][4];
#pragma unroll
  for (int mt = 0; mt < 8; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;

  int failed_at = -1;  // the stage whose wait gave up (CTA-uniform)
  for (int st = 0; st < n_st; ++st) {
    const int buf = st % kStages;
    const bool got = mbar_wait(smem_u32(&full_bar[buf]),
                               (uint32_t)(st / kStages) & 1u, &s_abort,
                               c.wait_ns);
    // Every thread takes the same branch, so the barriers below match.
    if (__syncthreads_or(got ? 0 : 1)) {
      if (tid == 0) {
        atomicOr(c.err, ERR_TIMEOUT);
        s_abort = 1;
      }
      failed_at = st;
      break;
    }
    unsigned char *K0 = smem + buf * kStageBytes, *K1 = K0 + kRows * 128;
    unsigned char *V0 = K0 + 2 * kRows * 128, *V1 = K0 + 3 * kRows * 128;
    const int base = st * kRows, t0 = warp * 16;
    {
      const int rn = m - base;  // the new row, if it is in this warp's tile
      if (rn >= t0 && rn < t0 + 16) {
        const int ch = lane & 15, half = ch >> 3, cc = ch & 7;
        const uint32_t off = rn * 128 + ((cc ^ (rn & 7)) << 4);
        unsigned char *dst = lane < 16 ? (half ? K1 : K0) : (half ? V1 : V0);
        const __nv_bfloat16 *src = (lane < 16 ? p.k_new : p.v_new) + krow * 128;
        *reinterpret_cast<int4 *>(dst + off) = reinterpret_cast<const int4 *>(src)[ch];
      }
      const int lo = max(t0, n - base);  // rows >= n: zero V (unset memory)
      for (int i = lane; i < (t0 + 16 - lo) * 16; i += 32) {
        const int r = lo + (i >> 4), c16 = i & 15;
        *reinterpret_cast<int4 *>((c16 < 8 ? V0 : V1) + r * 128 + (c16 & 7) * 16) =
            make_int4(0, 0, 0, 0);
      }
    }
    __syncwarp();
    if (base + t0 < n) {
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
      s[0] = ra < n ? (s[0] + s2[0]) * p.scale_log2e : -INFINITY;
      s[1] = ra < n ? (s[1] + s2[1]) * p.scale_log2e : -INFINITY;
      s[2] = rb < n ? (s[2] + s2[2]) * p.scale_log2e : -INFINITY;
      s[3] = rb < n ? (s[3] + s2[3]) * p.scale_log2e : -INFINITY;
      // keep the logits for the exact score update
      if (ra < n) {
        if (c2 < G) LG[c2 * nm + ra] = s[0];
        if (c2 + 1 < G) LG[(c2 + 1) * nm + ra] = s[1];
      }
      if (rb < n) {
        if (c2 < G) LG[c2 * nm + rb] = s[2];
        if (c2 + 1 < G) LG[(c2 + 1) * nm + rb] = s[3];
      }
      float x0 = fmaxf(s[0], s[2]), x1 = fmaxf(s[1], s[3]);
#pragma unroll
      for (int off = 4; off < 32; off <<= 1) {
        x0 = fmaxf(x0, __shfl_xor_sync(0xffffffffu, x0, off));
        x1 = fmaxf(x1, __shfl_xor_sync(0xffffffffu, x1, off));
      }
      const float n0 = fmaxf(m0, x0), n1 = fmaxf(m1, x1);
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
    fence_proxy_async();
    __syncthreads();
    if (tid == 0 && st + kStages < n_st) issue(st + kStages);
  }
  __syncthreads();
  if (failed_at >= 0) {
    // Stages failed_at .. failed_at + kStages - 1 (those below n_st) were
    // issued and not consumed: wait (bounded) for their copies to land.
    if (tid == 0) {
      volatile int never = 0;
      for (int st = failed_at; st < min(n_st, failed_at + kStages); ++st)
        mbar_wait(smem_u32(&full_bar[st % kStages]), (uint32_t)(st / kStages) & 1u,
                  &never);
    }
    return;
  }

  // Merge the warps: common max M and sum L per head, output rows.
#pragma unroll
  for (int off = 4; off < 32; off <<= 1) {
    l0 += __shfl_xor_sync(0xffffffffu, l0, off);
    l1 += __shfl_xor_sync(0xffffffffu, l1, off);
  }
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
  float *XO = reinterpret_cast<float *>(smem);  // stage buffers are free now
#pragma unroll
  for (int mt = 0; mt < 8; ++mt) {
    XO[((warp * 8 + mt) * 4 + 0) * 32 + lane] = o[mt][0] * f0;
    XO[((warp * 8 + mt) * 4 + 1) * 32 + lane] = o[mt][1] * f1;
    XO[((warp * 8 + mt) * 4 + 2) * 32 + lane] = o[mt][2] * f0;
    XO[((warp * 8 + mt) * 4 + 3) * 32 + lane] = o[mt][3] * f1;
  }
  if (lane < 4) {
    ML[kWarps * 8 + warp * 8 + c2] = l0 * f0;
    ML[kWarps * 8 + warp * 8 + c2 + 1] = l1 * f1;
  }
  __syncthreads();
  if (tid < 8) {  // per head: the merged max and 1 / sum
    float L = 0.f, M = -INFINITY;
    for (int w = 0; w < kWarps; ++w) {
      L += ML[kWarps * 8 + w * 8 + tid];
      M = fmaxf(M, ML[w * 8 + tid]);
    }
    ML[2 * kWarps * 8 + tid] = M;
    ML[2 * kWarps * 8 + 8 + tid] = 1.f / L;
    if (tid < G && !(L >= 1.f && L < INFINITY)) atomicOr(c.err, ERR_NONFINITE);
  }
  __syncthreads();
  const float *Mg = ML + 2 * kWarps * 8, *iLg = Mg + 8;
  {
    // out[g][d]: thread tid handles head-dim column pairs; fragment sums
    constexpr int osz = kOutBf16 ? 2 : 4;
    unsigned char *gout = reinterpret_cast<unsigned char *>(p.out) + krow * G * 128 * osz;
    for (int i = tid; i < 8 * 32 * 4; i += blockDim.x) {  // (mt, e, lane)
      const int ln = i & 31, e = (i >> 5) & 3, mt = i >> 7;
      float sum = 0.f;
#pragma unroll
      for (int w = 0; w < kWarps; ++w) sum += XO[((w * 8 + mt) * 4 + e) * 32 + ln];
      const int g = ((ln & 3) * 2) + (e & 1), d = 16 * mt + (ln >> 2) + 8 * (e >> 1);
      if (g < G) {
        const float v = sum * iLg[g];
        if (kOutBf16)
          reinterpret_cast<__nv_bfloat16 *>(gout)[g * 128 + d] = __float2bfloat16_rn(v);
        else
          reinterpret_cast<float *>(gout)[g * 128 + d] = v;
      }
    }
  }

  // Accumulated attention from the kept logits; the eviction candidate.
  const float inv_g = 1.f / (float)G;
  const int wlo = t - p.window;
  unsigned long long best = ~0ull;
  int bi = -1;
  for (int i = tid; i < n; i += blockDim.x) {
    float acc = 0.f;
    for (int g = 0; g < G; ++g) acc += exp2f(LG[g * nm + i] - Mg[g]) * iLg[g];
    const float s = (i < m ? SC[i] : 0.f) + acc * inv_g;
    NS[i] = s;
    const int pi = i < m ? PS[i] : t;
    if (pi <= wlo) {
      const unsigned long long key =
          ((unsigned long long)__float_as_uint(s) << 32) |
          (unsigned long long)(0xFFFFFFFFu - (unsigned)pi);
      if (key < best) {
        best = key;
        bi = i;
      }
    }
  }
  int victim = -1;
  if (p.evict && n > p.budget + p.window) {
#pragma unroll
    for (int o2 = 16; o2 > 0; o2 >>= 1) {
      const unsigned long long ob = __shfl_xor_sync(0xffffffffu, best, o2);
      const int oi = __shfl_xor_sync(0xffffffffu, bi, o2);
      if (ob < best) {
        best = ob;
        bi = oi;
      }
    }
    uint4 *RED = reinterpret_cast<uint4 *>(smem + Ly.red);
    if (lane == 0)
      RED[warp] = make_uint4((uint32_t)best, (uint32_t)(best >> 32), (uint32_t)bi, 0u);
    __syncthreads();
    for (int w = 0; w < kWarps; ++w) {
      const uint4 a = RED[w];
      const unsigned long long kb = ((unsigned long long)a.y << 32) | a.x;
      if (kb < best) {
        best = kb;
        bi = (int)a.z;
      }
    }
    victim = bi;
  }
  __syncthreads();

  // Write back: scores of the kept rows, the new row into the freed slot
  // (or the first free slot when nothing is evicted), length and position.
  float *gsc = c.score + ug * c.sstride;
  for (int i = tid; i < m; i += blockDim.x) gsc[i] = i == victim ? NS[m] : NS[i];
  const int slot = victim < 0 ? m : (victim < m ? victim : -1);
  if (slot >= 0 && tid < 32) {
    const int ch = tid & 15;
    __nv_bfloat16 *dst = reinterpret_cast<__nv_bfloat16 *>(tid < 16 ? c.K : c.V) +
                         (ug * (size_t)c.cap + slot) * 128;
    const __nv_bfloat16 *src = (tid < 16 ? p.k_new : p.v_new) + krow * 128;
    reinterpret_cast<int4 *>(dst)[ch] = reinterpret_cast<const int4 *>(src)[ch];
    if (tid == 0) {
      c.pos[ug * c.sstride + slot] = t;
      if (slot == m) gsc[m] = NS[m];
    }
  }
  if (tid == 0) {
    c.state[4 * ug] = victim < 0 ? m + 1 : m;
    c.state[4 * ug + 1] = t + 1;
    c.state[4 * ug + 2] = 0;  // the R-KV key sum no longer matches
  }
}

}  // namespace

int stream_box_rows() { return kBoxRows; }
int stream_max_rows() { return kMaxRowsStream; }
size_t stream_smem_bytes(int n_max) {
  return (size_t)StreamLayout(n_max).bytes + 1024;
}

cudaError_t launch_stream_step(const CUtensorMap &tmK, const CUtensorMap &tmV,
                               const StreamParams &p, cudaStream_t st) {
  const int smem = (int)stream_smem_bytes(p.n_max);
  const int units = p.c.S * p.nl * p.c.H;
  cudaError_t e;
  if (p.c.out_bf16) {
    e = cudaFuncSetAttribute(stream_step_kernel<true>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(stream_step_kernel<true>, dim3(units), dim3(32 * kWarps),
                      smem, st, tmK, tmV, p);
  } else {
    e = cudaFuncSetAttribute(stream_step_kernel<false>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(stream_step_kernel<false>, dim3(units), dim3(32 * kWarps),
                      smem, st, tmK, tmV, p);
  }
}

}  // namespace kvr
