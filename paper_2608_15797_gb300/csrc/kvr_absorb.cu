// kvr_absorb.cu -- absorbing a chunk of c tokens per (sequence, layer, KV
// head) in one launch: the base model's single forward pass over an accepted
// step (Algorithm 1) and prompt prefill that seeds the scores.  Token j is
// appended and attends every live row and the chunk's rows 0..j (causal);
// every token adds its head-mean probabilities to the accumulated scores of
// the rows it attends (Sec. 2.1); then the unit is cut back to B + W once
// (TopB of Eq. 1 with the window of Sec. 4.1).  bf16, head_dim 128, G <= 8,
// c <= 64, at most kMaxRows rows after the chunk.
//
// Design (GB300, sm_103a): one CTA of 8 warps per unit.
//  - The unit's live K/V rows and the chunk's new rows are copied into
//    shared memory (16-byte cp.async pieces, 128B-swizzled rows so ldmatrix
//    is conflict-free); every later read of K and V is from there.
//  - The c*G query rows are the M side of bf16 mma.sync (m16n8k16, fp32
//    accumulate): a warp takes 16 query rows at a time, their fragments
//    loaded straight from global memory.  Pass 1 runs QK^T over the rows
//    each query may see (causal bound) for the exact softmax statistics;
//    pass 2 recomputes QK^T, forms the exact probabilities, adds their
//    head-mean column sums to the unit's score accumulator (shared-memory
//    atomics) and runs PV with P split into two bf16 terms (hi + lo).
//  - The selection is a block radix select of the B-th best key among the
//    rows outside the window; survivors beyond B + W fill freed slots below
//    it, and new rows are written once, at their final slot, from shared
//    memory.
#include <cuda.h>
#include <cuda_bf16.h>
#include <math.h>
#include <stdint.h>

#include "kvr_device.cuh"
#include "kvr_internal.h"
#include "kvr_ptx.cuh"

namespace kvr {
namespace {

using namespace ptx;
using dev::kThreads;
using dev::kWarps;

constexpr int kMaxChunk = 64;
constexpr int kMaxRows = 192;
static_assert(kMaxRows <= kThreads, "one row per thread in the selection");

__device__ __forceinline__ void cp_async_commit_wait_all() {
  asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}

// Byte offset of 16-byte piece ch (0..15: columns 8ch..8ch+7) of row r
// within a K or V area: two 64-column halves of kRows rows, 128B swizzle.
__device__ __forceinline__ uint32_t swz(int r, int ch) {
  return (ch >> 3) * kMaxRows * 128 + r * 128 + (((ch & 7) ^ (r & 7)) << 4);
}

struct AbsorbSmem {
  static constexpr int k = 0;                          // [2][kMaxRows][128 B]
  static constexpr int v = k + 2 * kMaxRows * 128;     // same
  static constexpr int sc = v + 2 * kMaxRows * 128;    // old scores [kMaxRows]
  static constexpr int ps = sc + 4 * kMaxRows;         // positions
  static constexpr int acc = ps + 4 * kMaxRows;        // score increments
  static constexpr int lists = acc + 4 * kMaxRows;     // holes | movers
  static constexpr int key = lists + 8 * kMaxRows;     // selection keys
  static constexpr int kept = key + 8 * kMaxRows;      // kept flags
  static constexpr int bytes = kept + 4 * kMaxRows;
};

template <bool kOutBf16>
__global__ void __launch_bounds__(kThreads)
    absorb_kernel(const AbsorbParams p) {
  pdl_begin();
  extern __shared__ __align__(1024) unsigned char smem[];
  __shared__ int s_base, s_count;
  __shared__ int s_wsum[kWarps];
  const CacheView &c = p.c;
  const int G = c.G, C = p.chunk;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int idx = blockIdx.x;
  const int h = idx % c.H, lr = (idx / c.H) % p.nl, sq = idx / (c.H * p.nl);
  const size_t ug = ((size_t)sq * c.L + p.lb + lr) * c.H + h;
  const size_t row0 = ((size_t)sq * p.nl + lr) * C;  // token 0 of this row group
  const int n0 = c.state[4 * ug], t0 = c.state[4 * ug + 1];
  const int n = n0 + C;
  if (n0 < 0 || n > kMaxRows || n > c.cap) {
    if (tid == 0) atomicOr(c.err, n > c.cap ? ERR_CAPACITY : ERR_LENGTH);
    return;
  }
  __nv_bfloat16 *Ku = reinterpret_cast<__nv_bfloat16 *>(c.K) + ug * (size_t)c.cap * 128;
  __nv_bfloat16 *Vu = reinterpret_cast<__nv_bfloat16 *>(c.V) + ug * (size_t)c.cap * 128;
  float *su = c.score + ug * c.sstride;
  int32_t *pu = c.pos + ug * c.sstride;
  float *SC = reinterpret_cast<float *>(smem + AbsorbSmem::sc);
  int32_t *PS = reinterpret_cast<int32_t *>(smem + AbsorbSmem::ps);
  float *ACC = reinterpret_cast<float *>(smem + AbsorbSmem::acc);
  const uint32_t sK = smem_u32(smem + AbsorbSmem::k);
  const uint32_t sV = smem_u32(smem + AbsorbSmem::v);

  // Rows [0, n0) from the slab, rows n0 + j from the chunk's new k/v.
  for (int i = tid; i < n * 16; i += kThreads) {
    const int r = i >> 4, ch = i & 15;
    const __nv_bfloat16 *ks, *vs;
    if (r < n0) {
      ks = Ku + (size_t)r * 128;
      vs = Vu + (size_t)r * 128;
    } else {
      const size_t kr = (row0 + (r - n0)) * c.H + h;
      ks = p.k_new + kr * 128;
      vs = p.v_new + kr * 128;
    }
    cp_async16(sK + swz(r, ch), ks + ch * 8);
    cp_async16(sV + swz(r, ch), vs + ch * 8);
  }
  // V rows past n up to the end of their 16-row tile are read by PV with a
  // zero probability; zero them so stale bits (NaN) cannot leak in.
  for (int i = tid; i < (((n + 15) & ~15) - n) * 16; i += kThreads) {
    const int r = n + (i >> 4), ch = i & 15;
    *reinterpret_cast<int4 *>(smem + AbsorbSmem::v + swz(r, ch)) =
        make_int4(0, 0, 0, 0);
  }
  for (int r = tid; r < n; r += kThreads) {
    SC[r] = r < n0 ? su[r] : 0.f;
    PS[r] = r < n0 ? pu[r] : t0 + (r - n0);
    ACC[r] = 0.f;
  }
  cp_async_commit_wait_all();
  __syncthreads();

  // ---- attention: 16 query rows (token-major: row = j * G + g) per task ----
  const int MQ = C * G, n_tiles = (MQ + 15) / 16;
  const int r0l = lane >> 2, c2 = (lane & 3) * 2;
  const float inv_g = p.inv_g;
  for (int mt = warp; mt < n_tiles; mt += kWarps) {
    const int ra = mt * 16 + r0l, rb = ra + 8;  // this lane's two query rows
    const int ja = ra / G, jb = rb / G;
    const bool va = ra < MQ, vb = rb < MQ;
    // Causal bound: query row of token j sees key rows < n0 + j + 1.
    const int lim_a = va ? n0 + ja + 1 : 0, lim_b = vb ? n0 + jb + 1 : 0;
    const int lim_tile = n0 + min(C, (min(mt * 16 + 15, MQ - 1)) / G + 1);
    uint32_t qa[8][4];
    {
      const uint32_t *pa = va ? reinterpret_cast<const uint32_t *>(
                                    p.q + (((row0 + ja) * c.H + h) * G + ra % G) * 128)
                              : nullptr;
      const uint32_t *pb = vb ? reinterpret_cast<const uint32_t *>(
                                    p.q + (((row0 + jb) * c.H + h) * G + rb % G) * 128)
                              : nullptr;
#pragma unroll
      for (int ks = 0; ks < 8; ++ks) {
        const int e = 8 * ks + (lane & 3);  // 32-bit word of dims 16ks + 2t
        qa[ks][0] = va ? __ldg(pa + e) : 0u;
        qa[ks][1] = vb ? __ldg(pb + e) : 0u;
        qa[ks][2] = va ? __ldg(pa + e + 4) : 0u;
        qa[ks][3] = vb ? __ldg(pb + e + 4) : 0u;
      }
    }
    // S tile for key rows [kt*16, kt*16 + 16): two n8 halves, scaled log2.
    auto logits = [&](int kt, float (&s)[2][4]) {
      float s2[2][4];  // odd k-steps on a second chain
#pragma unroll
      for (int hf = 0; hf < 2; ++hf)
        s[hf][0] = s[hf][1] = s[hf][2] = s[hf][3] = s2[hf][0] = s2[hf][1] =
            s2[hf][2] = s2[hf][3] = 0.f;
      const int kr = kt * 16 + (lane & 7) + ((lane >> 4) << 3);
#pragma unroll
      for (int ks = 0; ks < 8; ++ks) {
        const int ch = 2 * ks + ((lane >> 3) & 1);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(sK + swz(kr, ch), b0, b1, b2, b3);
        float(&t)[2][4] = (ks & 1) ? s2 : s;
        mma_bf16(t[0], qa[ks][0], qa[ks][1], qa[ks][2], qa[ks][3], b0, b1);
        mma_bf16(t[1], qa[ks][0], qa[ks][1], qa[ks][2], qa[ks][3], b2, b3);
      }
#pragma unroll
      for (int hf = 0; hf < 2; ++hf)
#pragma unroll
        for (int e = 0; e < 4; ++e) s[hf][e] += s2[hf][e];
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
        const int col = kt * 16 + hf * 8 + c2;
        s[hf][0] = col < lim_a ? s[hf][0] * p.scale_log2e : -INFINITY;
        s[hf][1] = col + 1 < lim_a ? s[hf][1] * p.scale_log2e : -INFINITY;
        s[hf][2] = col < lim_b ? s[hf][2] * p.scale_log2e : -INFINITY;
        s[hf][3] = col + 1 < lim_b ? s[hf][3] * p.scale_log2e : -INFINITY;
      }
    };
    const int n_kt = (lim_tile + 15) / 16;
    // Pass 1: row maxima and sums (online over key tiles).
    float ma = -INFINITY, mb = -INFINITY, la = 0.f, lb = 0.f;
    for (int kt = 0; kt < n_kt; ++kt) {
      float s[2][4];
      logits(kt, s);
      float xa = fmaxf(fmaxf(s[0][0], s[0][1]), fmaxf(s[1][0], s[1][1]));
      float xb = fmaxf(fmaxf(s[0][2], s[0][3]), fmaxf(s[1][2], s[1][3]));
      xa = fmaxf(xa, __shfl_xor_sync(0xffffffffu, xa, 1));
      xa = fmaxf(xa, __shfl_xor_sync(0xffffffffu, xa, 2));
      xb = fmaxf(xb, __shfl_xor_sync(0xffffffffu, xb, 1));
      xb = fmaxf(xb, __shfl_xor_sync(0xffffffffu, xb, 2));
      const float na = fmaxf(ma, xa), nb = fmaxf(mb, xb);
      // A row whose keys so far are all masked keeps max -inf: no terms yet.
      const float ua = na == -INFINITY ? 0.f : na, ub = nb == -INFINITY ? 0.f : nb;
      float pa = ex2(s[0][0] - ua) + ex2(s[0][1] - ua) + ex2(s[1][0] - ua) + ex2(s[1][1] - ua);
      float pb = ex2(s[0][2] - ub) + ex2(s[0][3] - ub) + ex2(s[1][2] - ub) + ex2(s[1][3] - ub);
      pa += __shfl_xor_sync(0xffffffffu, pa, 1);
      pa += __shfl_xor_sync(0xffffffffu, pa, 2);
      pb += __shfl_xor_sync(0xffffffffu, pb, 1);
      pb += __shfl_xor_sync(0xffffffffu, pb, 2);
      la = (ma == -INFINITY ? 0.f : la * ex2(ma - ua)) + pa;
      lb = (mb == -INFINITY ? 0.f : lb * ex2(mb - ub)) + pb;
      ma = na;
      mb = nb;
    }
    const float ia = va ? rcp(la) : 0.f, ib = vb ? rcp(lb) : 0.f;
    // Padding rows (past c * G) have no live key: reference 0, probability 0.
    if (!va) ma = 0.f;
    if (!vb) mb = 0.f;
    if (va && lane == 0 && !(la > 0.5f && la < INFINITY)) atomicOr(c.err, ERR_NONFINITE);
    // Pass 2: exact probabilities, score increments, PV.
    float o[16][4];
#pragma unroll
    for (int nt = 0; nt < 16; ++nt) o[nt][0] = o[nt][1] = o[nt][2] = o[nt][3] = 0.f;
    for (int kt = 0; kt < n_kt; ++kt) {
      float s[2][4];
      logits(kt, s);
      float pr[2][4];
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
        pr[hf][0] = ex2(s[hf][0] - ma) * ia;
        pr[hf][1] = ex2(s[hf][1] - ma) * ia;
        pr[hf][2] = ex2(s[hf][2] - mb) * ib;
        pr[hf][3] = ex2(s[hf][3] - mb) * ib;
        // Column sums over the 16 query rows (lanes sharing lane % 4).
        float x0 = pr[hf][0] + pr[hf][2], x1 = pr[hf][1] + pr[hf][3];
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) {
          x0 += __shfl_xor_sync(0xffffffffu, x0, off);
          x1 += __shfl_xor_sync(0xffffffffu, x1, off);
        }
        const int col = kt * 16 + hf * 8 + c2;
        if (lane < 4) {
          if (col < n) atomicAdd(&ACC[col], x0 * inv_g);
          if (col + 1 < n) atomicAdd(&ACC[col + 1], x1 * inv_g);
        }
      }
      // P as the A operand (rows = query rows, k = the tile's 16 key rows),
      // hi and lo bf16 terms.
      uint32_t ph[4], pl[4];
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
        const uint32_t h0 = pack_bf16(pr[hf][0], pr[hf][1]);
        const uint32_t h1 = pack_bf16(pr[hf][2], pr[hf][3]);
        const __nv_bfloat162 b0 = *reinterpret_cast<const __nv_bfloat162 *>(&h0);
        const __nv_bfloat162 b1 = *reinterpret_cast<const __nv_bfloat162 *>(&h1);
        ph[2 * hf] = h0;
        ph[2 * hf + 1] = h1;
        pl[2 * hf] = pack_bf16(pr[hf][0] - __low2float(b0), pr[hf][1] - __high2float(b0));
        pl[2 * hf + 1] = pack_bf16(pr[hf][2] - __low2float(b1), pr[hf][3] - __high2float(b1));
      }
      const int vr = kt * 16 + (lane & 7) + (((lane >> 3) & 1) << 3);
#pragma unroll
      for (int dp = 0; dp < 8; ++dp) {  // 16 head-dim columns per ldmatrix
        const int ch = 2 * dp + (lane >> 4);
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(sV + swz(vr, ch), b0, b1, b2, b3);
        mma_bf16(o[2 * dp], ph[0], ph[1], ph[2], ph[3], b0, b1);
        mma_bf16(o[2 * dp], pl[0], pl[1], pl[2], pl[3], b0, b1);
        mma_bf16(o[2 * dp + 1], ph[0], ph[1], ph[2], ph[3], b2, b3);
        mma_bf16(o[2 * dp + 1], pl[0], pl[1], pl[2], pl[3], b2, b3);
      }
    }
    // Output rows (token j, head g): columns 8 nt + c2, + 1.
    constexpr int osz = kOutBf16 ? 2 : 4;
#pragma unroll
    for (int hs = 0; hs < 2; ++hs) {
      const int r = hs ? rb : ra;
      if (r >= MQ) continue;
      const int j = r / G, g = r % G;
      unsigned char *orow = reinterpret_cast<unsigned char *>(p.out) +
                            ((((row0 + j) * c.H + h) * G + g) * 128) * osz;
#pragma unroll
      for (int nt = 0; nt < 16; ++nt) {
        const float x = o[nt][2 * hs], y = o[nt][2 * hs + 1];
        if (kOutBf16)
          *reinterpret_cast<uint32_t *>(orow + (8 * nt + c2) * 2) = pack_bf16(x, y);
        else
          *reinterpret_cast<float2 *>(orow + (8 * nt + c2) * 4) = make_float2(x, y);
      }
    }
  }
  __syncthreads();

  // ---- scores, selection, compaction ----
  for (int r = tid; r < n; r += kThreads) SC[r] += ACC[r];
  __syncthreads();
  const int B = p.budget, W = p.window;
  const bool cut = p.evict && n > B + W;
  const int wlo = t0 + C - 1 - W;  // a row is a candidate iff pos <= wlo
  // TopB by rank (n <= kMaxRows <= kThreads rows, one per thread): a
  // candidate stays iff fewer than B candidates have a larger key (keys are
  // distinct: positions are).  Rows outside the window-free set always stay.
  unsigned long long *KEY = reinterpret_cast<unsigned long long *>(smem + AbsorbSmem::key);
  int *KEPT = reinterpret_cast<int *>(smem + AbsorbSmem::kept);
  for (int r = tid; r < n; r += kThreads)
    KEY[r] = PS[r] <= wlo ? dev::rank_key(SC[r], PS[r]) : 0ull;
  __syncthreads();
  for (int r = tid; r < n; r += kThreads) {
    int k = 1;
    if (cut && PS[r] <= wlo) {
      const unsigned long long mine_key = KEY[r];
      int above = 0;
      for (int j = 0; j < n; ++j) above += KEY[j] > mine_key ? 1 : 0;
      k = above < B ? 1 : 0;
    }
    KEPT[r] = k;
  }
  __syncthreads();
  auto keep = [&](int i) { return KEPT[i] != 0; };
  if (tid == 0) s_count = 0;
  __syncthreads();
  int mine = 0;
  for (int i = tid; i < n; i += kThreads) mine += keep(i) ? 1 : 0;
  atomicAdd(&s_count, mine);
  __syncthreads();
  const int nk = s_count;
  if (cut && nk != B + W) {
    if (tid == 0) atomicOr(c.err, ERR_LENGTH);
    return;
  }
  int *lists = reinterpret_cast<int *>(smem + AbsorbSmem::lists);
  int *holes = lists, *movers = lists + kMaxRows;
  const int nh = dev::block_collect(0, nk, [&](int i) { return !keep(i); }, holes,
                                    s_wsum, &s_base);
  const int nm = dev::block_collect(nk, n, keep, movers, s_wsum, &s_base);
  if (nh != nm) {
    if (tid == 0) atomicOr(c.err, ERR_LENGTH);
    return;
  }
  // Final slot of every kept row: its own below nk, a hole for a mover.
  // Rows whose bytes must be written: new rows (r >= n0) that stay below nk,
  // and every mover (all rows are in shared memory).
  auto write_row = [&](int src, int dst, int ln) {  // one warp-lane share
    const int ch = ln & 15;
    const uint32_t from = (ln < 16 ? sK : sV) + swz(src, ch);
    int4 val;
    asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(val.x), "=r"(val.y), "=r"(val.z), "=r"(val.w)
                 : "r"(from));
    __nv_bfloat16 *base = ln < 16 ? Ku : Vu;
    reinterpret_cast<int4 *>(base + (size_t)dst * 128)[ch] = val;
  };
  for (int r = n0 + warp; r < nk; r += kWarps)  // new rows kept in place
    if (keep(r)) write_row(r, r, lane);
  for (int k = warp; k < nh; k += kWarps) write_row(movers[k], holes[k], lane);
  for (int r = tid; r < nk; r += kThreads)
    if (keep(r)) {
      su[r] = SC[r];
      pu[r] = PS[r];
    }
  for (int k = tid; k < nh; k += kThreads) {
    su[holes[k]] = SC[movers[k]];
    pu[holes[k]] = PS[movers[k]];
  }
  if (tid == 0) {
    c.state[4 * ug] = nk;
    c.state[4 * ug + 1] = t0 + C;
  }
}

}  // namespace

int absorb_max_chunk() { return kMaxChunk; }
int absorb_max_rows() { return kMaxRows; }

cudaError_t launch_absorb(const AbsorbParams &p, cudaStream_t st) {
  if (p.chunk < 1 || p.chunk > kMaxChunk || p.c.G > 8 || p.c.d != 128 ||
      !p.c.kv_bf16)
    return cudaErrorInvalidValue;
  const int units = p.c.S * p.nl * p.c.H;
  const int smem = AbsorbSmem::bytes;
  auto kern = p.c.out_bf16 ? absorb_kernel<true> : absorb_kernel<false>;
  cudaError_t e = cudaFuncSetAttribute(
      kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(kern, dim3(units), dim3(kThreads), (size_t)smem, st, p);
}

}  // namespace kvr
