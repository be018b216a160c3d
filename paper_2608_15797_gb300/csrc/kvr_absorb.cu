// kvr_absorb.cu -- absorbing a chunk of c tokens per (sequence, layer, KV
// head) in one launch: the base model's single forward pass over an accepted
// step (Algorithm 1) and prompt prefill that seeds the scores.  Token j is
// appended and attends every live row and the chunk's rows 0..j (causal);
// every token adds its head-mean probabilities to the accumulated scores of
// the rows it attends (Sec. 2.1); then the unit is cut back to B + W once
// (TopB of Eq. 1 with the window of Sec. 4.1).  bf16, head_dim 128, G <= 8,
// c <= 64, at most kMaxRows rows after the chunk.
//
// Design (GB300, sm_103a): one CTA of 8 warps per unit, in two kernels
// that share the load and the selection.  absorb_tc_kernel (5th-generation
// tensor cores, two CTAs an SM; described before it) takes units of at most
// 144 rows after the chunk; absorb_kernel (mma.sync) takes the rest, up to
// kMaxRows, or any unit when selected.
//  - The unit's live K/V rows and the chunk's new rows are copied into
//    shared memory (16-byte cp.async pieces, 128B-swizzled rows so ldmatrix
//    and the tensor-core descriptors read them conflict-free); every later
//    read of K and V is from there.
//  - absorb_kernel: the c*G query rows are the M side of bf16 mma.sync (m16n8k16, fp32
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

// Packed fp32 pairs (round to nearest, no flush: the scalar code's results).
__device__ __forceinline__ uint64_t pk2(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void upk2(uint64_t v, float &lo, float &hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t add2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ uint64_t mul2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

__device__ __forceinline__ void cp_async_commit_wait_all() {
  asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}

// Byte offset of 16-byte piece ch (0..15: columns 8ch..8ch+7) of row r
// within a K or V area: two 64-column halves of kRows rows, 128B swizzle.
template <int kRows>
__device__ __forceinline__ uint32_t swzr(int r, int ch) {
  return (ch >> 3) * kRows * 128 + r * 128 + (((ch & 7) ^ (r & 7)) << 4);
}
__device__ __forceinline__ uint32_t swz(int r, int ch) { return swzr<kMaxRows>(r, ch); }

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

// The unit a CTA absorbs into, and where its arrays live in shared memory.
struct Unit {
  size_t ug, row0;
  int h, n0, t0, n;
  __nv_bfloat16 *Ku, *Vu;
  float *su;
  int32_t *pu;
};
struct UnitSmem {
  unsigned char *k, *v;
  float *sc, *acc;
  int32_t *ps;
  int *lists;
  unsigned long long *key;
  int *kept;
};

__device__ __forceinline__ bool unit_begin(const AbsorbParams &p, Unit &u,
                                           int max_rows = kMaxRows) {
  const CacheView &c = p.c;
  const int idx = blockIdx.x;
  u.h = idx % c.H;
  const int lr = (idx / c.H) % p.nl, sq = idx / (c.H * p.nl);
  u.ug = ((size_t)sq * c.L + p.lb + lr) * c.H + u.h;
  u.row0 = ((size_t)sq * p.nl + lr) * p.chunk;  // token 0 of this row group
  u.n0 = c.state[4 * u.ug];
  u.t0 = c.state[4 * u.ug + 1];
  u.n = u.n0 + p.chunk;
  if (u.n0 < 0 || u.n > max_rows || u.n > c.cap) {
    if (threadIdx.x == 0) atomicOr(c.err, u.n > c.cap ? ERR_CAPACITY : ERR_LENGTH);
    return false;
  }
  u.Ku = reinterpret_cast<__nv_bfloat16 *>(c.K) + u.ug * (size_t)c.cap * 128;
  u.Vu = reinterpret_cast<__nv_bfloat16 *>(c.V) + u.ug * (size_t)c.cap * 128;
  u.su = c.score + u.ug * c.sstride;
  u.pu = c.pos + u.ug * c.sstride;
  return true;
}

// Rows [0, n0) from the slab, rows n0 + j from the chunk's new k/v (K and V
// areas of kRows rows per 64-column half); scores, positions and zeroed
// increments.  Ends with the CTA synchronised.
template <int kRows = kMaxRows>
__device__ void load_unit(const AbsorbParams &p, const Unit &u,
                          const UnitSmem &m) {
  const CacheView &c = p.c;
  const int tid = threadIdx.x, n = u.n, n0 = u.n0;
  const uint32_t sK = smem_u32(m.k), sV = smem_u32(m.v);
  for (int i = tid; i < n * 16; i += kThreads) {
    const int r = i >> 4, ch = i & 15;
    const __nv_bfloat16 *ks, *vs;
    if (r < n0) {
      ks = u.Ku + (size_t)r * 128;
      vs = u.Vu + (size_t)r * 128;
    } else {
      const size_t kr = (u.row0 + (r - n0)) * c.H + u.h;
      ks = p.k_new + kr * 128;
      vs = p.v_new + kr * 128;
    }
    cp_async16(sK + swzr<kRows>(r, ch), ks + ch * 8);
    cp_async16(sV + swzr<kRows>(r, ch), vs + ch * 8);
  }
  // V rows past n up to the end of their 16-row tile are read by PV with a
  // zero probability; zero them so stale bits (NaN) cannot leak in.
  for (int i = tid; i < (((n + 15) & ~15) - n) * 16; i += kThreads) {
    const int r = n + (i >> 4), ch = i & 15;
    *reinterpret_cast<int4 *>(m.v + swzr<kRows>(r, ch)) = make_int4(0, 0, 0, 0);
  }
  for (int r = tid; r < n; r += kThreads) {
    m.sc[r] = r < n0 ? u.su[r] : 0.f;
    m.ps[r] = r < n0 ? u.pu[r] : u.t0 + (r - n0);
    m.acc[r] = 0.f;
  }
  cp_async_commit_wait_all();
  fence_proxy_async();  // the rows are read by the tensor cores' async proxy too
  __syncthreads();
}

// Scores, the TopB cut and compaction, then the unit's state (K and V areas
// and row lists of kRows rows).
template <int kRows = kMaxRows>
__device__ void finish_unit(const AbsorbParams &p, const Unit &u,
                            const UnitSmem &m, int *s_wsum) {
  const CacheView &c = p.c;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int n = u.n, n0 = u.n0, C = p.chunk;
  float *SC = m.sc;
  int32_t *PS = m.ps;
  static_assert(kRows <= kThreads, "one thread a row");
  const int B = p.budget, W = p.window;
  const bool cut = p.evict && n > B + W;
  const int wlo = u.t0 + C - 1 - W;  // a row is a candidate iff pos <= wlo
  // Thread t owns row t: its final score and its TopB key.
  const int row = tid;
  const bool live = row < n;
  unsigned long long *KEY = m.key;
  int *KEPT = m.kept;
  if (live) {
    SC[row] += m.acc[row];
    KEY[row] = PS[row] <= wlo ? dev::rank_key(SC[row], PS[row]) : 0ull;
  }
  __syncthreads();
  // TopB by rank: a candidate stays iff fewer than B candidates have a
  // larger key (keys are distinct: positions are).  Rows outside the
  // window-free set always stay.
  bool kp = live;
  if (live && cut && PS[row] <= wlo) {
    const unsigned long long mine_key = KEY[row];
    int above = 0;
#pragma unroll 4
    for (int j = 0; j < n; ++j) above += KEY[j] > mine_key ? 1 : 0;
    kp = above < B;
  }
  if (live) KEPT[row] = kp ? 1 : 0;
  // Kept count, then the holes below it and the movers above it, each from
  // warp ballots and a prefix over the warps' counts.
  int *s_nk = s_wsum, *s_nh = s_wsum + kWarps, *s_nm = s_wsum + 2 * kWarps;
  const unsigned below = (1u << lane) - 1u;
  const unsigned bk = __ballot_sync(0xffffffffu, kp);
  if (lane == 0) s_nk[warp] = __popc(bk);
  __syncthreads();
  int nk = 0;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) nk += s_nk[w];
  if (cut && nk != B + W) {
    if (tid == 0) atomicOr(c.err, ERR_LENGTH);
    return;
  }
  const bool is_hole = live && row < nk && !kp, is_mover = live && row >= nk && kp;
  const unsigned bh = __ballot_sync(0xffffffffu, is_hole);
  const unsigned bm = __ballot_sync(0xffffffffu, is_mover);
  if (lane == 0) {
    s_nh[warp] = __popc(bh);
    s_nm[warp] = __popc(bm);
  }
  __syncthreads();
  int oh = 0, om = 0, nh = 0, nm = 0;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) {
    oh += w < warp ? s_nh[w] : 0;
    om += w < warp ? s_nm[w] : 0;
    nh += s_nh[w];
    nm += s_nm[w];
  }
  int *holes = m.lists, *movers = m.lists + kRows;
  if (is_hole) holes[oh + __popc(bh & below)] = row;
  if (is_mover) movers[om + __popc(bm & below)] = row;
  if (nh != nm) {
    if (tid == 0) atomicOr(c.err, ERR_LENGTH);
    return;
  }
  __syncthreads();
  auto keep = [&](int i) { return KEPT[i] != 0; };
  // Final slot of every kept row: its own below nk, a hole for a mover.
  // Rows whose bytes must be written: new rows (r >= n0) that stay below nk,
  // and every mover (all rows are in shared memory).
  const uint32_t sK = smem_u32(m.k), sV = smem_u32(m.v);
  auto write_row = [&](int src, int dst, int ln) {  // one warp-lane share
    const int ch = ln & 15;
    const uint32_t from = (ln < 16 ? sK : sV) + swzr<kRows>(src, ch);
    int4 val;
    asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(val.x), "=r"(val.y), "=r"(val.z), "=r"(val.w)
                 : "r"(from));
    __nv_bfloat16 *base = ln < 16 ? u.Ku : u.Vu;
    reinterpret_cast<int4 *>(base + (size_t)dst * 128)[ch] = val;
  };
  for (int r = n0 + warp; r < nk; r += kWarps)  // new rows kept in place
    if (keep(r)) write_row(r, r, lane);
  for (int k = warp; k < nh; k += kWarps) write_row(movers[k], holes[k], lane);
  for (int r = tid; r < nk; r += kThreads)
    if (keep(r)) {
      u.su[r] = SC[r];
      u.pu[r] = PS[r];
    }
  for (int k = tid; k < nh; k += kThreads) {
    u.su[holes[k]] = SC[movers[k]];
    u.pu[holes[k]] = PS[movers[k]];
  }
  if (tid == 0) {
    c.state[4 * u.ug] = nk;
    c.state[4 * u.ug + 1] = u.t0 + C;
    c.state[4 * u.ug + 2] = 0;  // the R-KV key sum no longer matches
  }
}

template <bool kOutBf16>
__global__ void __launch_bounds__(kThreads)
    absorb_kernel(const AbsorbParams p) {
  pdl_begin();
  extern __shared__ __align__(1024) unsigned char smem[];
  __shared__ int s_wsum[3 * kWarps];  // per-warp counts for the selection
  const CacheView &c = p.c;
  const int G = c.G, C = p.chunk;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  Unit u;
  if (!unit_begin(p, u)) return;
  const UnitSmem m{smem + AbsorbSmem::k,
                   smem + AbsorbSmem::v,
                   reinterpret_cast<float *>(smem + AbsorbSmem::sc),
                   reinterpret_cast<float *>(smem + AbsorbSmem::acc),
                   reinterpret_cast<int32_t *>(smem + AbsorbSmem::ps),
                   reinterpret_cast<int *>(smem + AbsorbSmem::lists),
                   reinterpret_cast<unsigned long long *>(smem + AbsorbSmem::key),
                   reinterpret_cast<int *>(smem + AbsorbSmem::kept)};
  load_unit(p, u, m);
  const int n = u.n, n0 = u.n0, h = u.h;
  const size_t row0 = u.row0;
  float *ACC = m.acc;
  const uint32_t sK = smem_u32(m.k), sV = smem_u32(m.v);
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

  finish_unit(p, u, m, s_wsum);
}

// ---- the same absorb on 5th-generation tensor cores ------------------------
//
// Units of at most kTcMaxRows rows after the chunk, two CTAs an SM (about
// 114 KB of shared memory and 256 tensor-memory columns each), so that one
// unit's loads, selection and stores overlap the other's tensor work.
// Query rows go in tiles of 128 / G whole tokens (row token * G + g; M =
// 128), with the unit's keys as N and K = the head dimension.  Per tile:
//   1. The tile's q rows arrive by TMA (one 4-D box per 64-column half,
//      K-major, 128B swizzle; the next tile's are fetched once this tile's
//      S is done) and thread 32 issues S = Q K^T into tensor memory (fp32;
//      N = the tile's causal limit rounded up to 16 keys).
//   2. Every warp reads its rows' logits from tensor memory once; warps w
//      and w + 4 share TMEM lanes 32 (w % 4).. and take half the columns
//      each.  They form the row statistics (an exchange on a named barrier
//      per pair), then the exact probabilities: P in place of the logits
//      (each 16-key chunk's 16 columns take its 8 hi and 8 lo columns of
//      bf16 pairs, the A operand of PV), and their column sums over the
//      warp's 32 rows (a shuffle butterfly into one slot per lane quarter,
//      summed in a fixed order) for the scores.  Chunks past a warp's last
//      causal limit are neither read nor exponentiated.
//   3. Thread 0 issues O = P_hi V + P_lo V one 64-column half of the head
//      dimension at a time (64 tensor-memory columns); the second half's
//      MMAs start once every thread has read the first, and the next
//      tile's S once the second half is done.
// Every mbarrier wait is bounded; tensor memory is freed before the
// selection.
constexpr int kTcMaxRows = 144;                    // rows this kernel stages
constexpr int kTcRows = 128;                       // query rows per tile
constexpr uint32_t kTcS = 0;                       // TMEM columns: S / P
constexpr uint32_t kTcO = kTcMaxRows;              //   O, one 64-column half
constexpr int kTcCols = 256;
constexpr int kTcChunks = (kTcMaxRows / 2 + 15) / 16;  // a thread's column chunks
static_assert(kTcO + 64 <= kTcCols, "TMEM columns");
static_assert(kTcMaxRows % 16 == 0, "whole 16-key chunks");

struct TcSmem {  // offsets from a 1024-byte aligned base
  static constexpr int k = 0;                              // [2][kTcMaxRows][128 B]
  static constexpr int v = k + 2 * kTcMaxRows * 128;
  static constexpr int q = v + 2 * kTcMaxRows * 128;       // [2][128][128 B]
  static constexpr int sc = q + 2 * kTcRows * 128;
  static constexpr int ps = sc + 4 * kTcMaxRows;
  static constexpr int acc = ps + 4 * kTcMaxRows;
  static constexpr int lists = acc + 4 * kTcMaxRows;
  static constexpr int key = lists + 8 * kTcMaxRows;       // also the (max, sum) exchange
  static constexpr int kept = key + 8 * kTcMaxRows;
  static constexpr int part = kept + 4 * kTcMaxRows;        // [4][kTcMaxRows] column sums
  static constexpr int bytes = part + 16 * kTcMaxRows;
  static constexpr int alloc = bytes + 1024;               // room to align
};
static_assert(8 * kTcMaxRows >= 8 * kTcRows, "the exchange fits in the key and list areas");
// Two CTAs an SM: 228 KB less 1 KB reserved per CTA, with room for the
// static variables.
static_assert(TcSmem::alloc + 512 <= 113 * 1024, "two CTAs an SM");

// Column sums of v[16] (this lane's row) over the warp's 32 rows: after the
// butterfly, lane l holds the sum of column (l >> 1) & 15... in the order
// below; both lanes of a pair hold the same value.  Returns the column.
__device__ __forceinline__ float colsum32(const float (&v)[16], int lane, int &col) {
  float a[8], b[4], cc[2];
  const bool b4 = (lane & 16) != 0, b3 = (lane & 8) != 0, b2 = (lane & 4) != 0,
             b1 = (lane & 2) != 0;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const float send = b4 ? v[i] : v[i + 8], keep = b4 ? v[i + 8] : v[i];
    a[i] = keep + __shfl_xor_sync(0xffffffffu, send, 16);
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float send = b3 ? a[i] : a[i + 4], keep = b3 ? a[i + 4] : a[i];
    b[i] = keep + __shfl_xor_sync(0xffffffffu, send, 8);
  }
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const float send = b2 ? b[i] : b[i + 2], keep = b2 ? b[i + 2] : b[i];
    cc[i] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
  }
  const float send = b1 ? cc[0] : cc[1], keep = b1 ? cc[1] : cc[0];
  float x = keep + __shfl_xor_sync(0xffffffffu, send, 2);
  x += __shfl_xor_sync(0xffffffffu, x, 1);
  col = (b4 ? 8 : 0) + (b3 ? 4 : 0) + (b2 ? 2 : 0) + (b1 ? 1 : 0);
  return x;
}

__device__ __forceinline__ void mma_ts_all(uint32_t d, uint32_t a, uint64_t b, uint32_t id,
                                           bool acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d),
      "r"(a), "l"(b), "r"(id), "r"(acc ? 1 : 0)
      : "memory");
}
__device__ __forceinline__ void tmem_st8(uint32_t taddr, const uint32_t (&v)[8]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"r"(taddr),
      "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]),
      "r"(v[7])
      : "memory");
}

template <bool kOutBf16>
__global__ void __launch_bounds__(kThreads, 2)
    absorb_tc_kernel(const AbsorbParams p, const __grid_constant__ CUtensorMap tmQ) {
  pdl_begin();
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  __shared__ int s_wsum[3 * kWarps];  // per-warp counts for the selection
  __shared__ uint32_t s_tmem;
  __shared__ int s_abort;
  __shared__ int s_q;  // thread 32's q state: bit 0 the phase to wait, bit 1 a load in flight
  __shared__ int s_dq[4];  // (32 q4 + 31) / G: the last token of rows 32 q4 .. 32 q4 + 31
  __shared__ __align__(8) uint64_t bar_s, bar_o, bar_q;
  unsigned char *smem = smem_raw + ((1024 - (smem_u32(smem_raw) & 1023)) & 1023);
  const CacheView &c = p.c;
  const int G = c.G, C = p.chunk;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  Unit u;
  if (!unit_begin(p, u, kTcMaxRows)) return;
  const UnitSmem m{smem + TcSmem::k,
                   smem + TcSmem::v,
                   reinterpret_cast<float *>(smem + TcSmem::sc),
                   reinterpret_cast<float *>(smem + TcSmem::acc),
                   reinterpret_cast<int32_t *>(smem + TcSmem::ps),
                   reinterpret_cast<int *>(smem + TcSmem::lists),
                   reinterpret_cast<unsigned long long *>(smem + TcSmem::key),
                   reinterpret_cast<int *>(smem + TcSmem::kept)};
  // The (max, sum) exchange of the lower and the upper warps, in areas the
  // selection uses only after the tiles.
  float2 *s_ml = reinterpret_cast<float2 *>(smem + TcSmem::key);
  float2 *s_mh = reinterpret_cast<float2 *>(smem + TcSmem::lists);
  if (warp == 0) tmem_alloc(smem_u32(&s_tmem), kTcCols);
  const int n = u.n, n0 = u.n0, h = u.h;
  const uint32_t aQ = smem_u32(smem + TcSmem::q);
  // Tile mt holds tokens [mt Jt, mt Jt + Jt) of the chunk (Jt = 128 / G
  // whole tokens) as rows token * G + g: one TMA box {64, G, 1, Jt} per
  // 64-column half, 128-byte swizzle.  Rows past Jt G keep what they held
  // and rows past the chunk hold other units' queries (or zeros past the
  // tensor); both are masked below.
  const int Jt = kTcRows / G, n_mt = (C + Jt - 1) / Jt;
  const uint32_t q_bytes = 256u * (uint32_t)(G * Jt);
  auto load_q = [&](int mt) {  // one thread
    mbar_expect_tx(smem_u32(&bar_q), q_bytes);
    for (int hf = 0; hf < 2; ++hf)
      tma_load_4d(aQ + hf * (kTcRows * 128), &tmQ, 64 * hf, 0, h, (int)u.row0 + mt * Jt,
                  smem_u32(&bar_q));
  };
  if (tid < 4) s_dq[tid] = (32 * tid + 31) / G;
  if (tid == 32) {
    mbar_init(smem_u32(&bar_s), 1);
    mbar_init(smem_u32(&bar_o), 1);
    mbar_init(smem_u32(&bar_q), 1);
    s_abort = 0;
    s_q = 2;
    fence_mbar_init();
    load_q(0);
  }
  tc_fence_before();
  load_unit<kTcMaxRows>(p, u, m);  // ends with the copies complete, the async proxy fenced and a barrier
  tc_fence_after();
  const uint32_t tm = s_tmem;
  const uint32_t aK = smem_u32(m.k), aV = smem_u32(m.v);
  const int wq = warp & 3;             // TMEM lane quarter of this warp
  const bool upper = warp >= 4;        // second half of the tile's columns
  const int r = wq * 32 + lane;        // this thread's row of the tile
  const uint32_t trow = tm + ((uint32_t)(wq * 32) << 16);
  const float scale = p.scale_log2e, inv_g = p.inv_g;
  float *ACC = m.acc;
  float *PART = reinterpret_cast<float *>(smem + TcSmem::part);
  volatile int *abort = &s_abort;
  // Keys that rows 32 q4 .. 32 q4 + 31 of tile mt may see: the causal
  // limit of the last of them below the tile's valid rows, 0 when there is
  // none.
  auto lim_warp = [&](int mt, int q4) {
    const int toks = min(Jt, C - mt * Jt);  // the tile's tokens
    if (32 * q4 >= toks * G) return 0;
    return n0 + mt * Jt + min(s_dq[q4], toks - 1) + 1;
  };
  // Columns of S tile mt: its keys rounded up to whole 16-key chunks
  // (P is zero past the last row's limit, so no MMA reads further).
  auto tile_cols = [&](int mt) { return (n0 + min(mt * Jt + Jt, C) + 15) & ~15; };
  // MMA issue, one thread each (S: thread 32; PV: thread 0).
  auto issue_s = [&](int mt) {
    const uint32_t id_s = idesc_bf16(kTcRows, tile_cols(mt), false);
#pragma unroll
    for (int k = 0; k < 8; ++k) {  // K = 128 head-dim columns, 16 a step
      const uint32_t off = (k & 3) * 32;
      tc_mma(tm + kTcS, sdesc_sw128(aQ + (k >> 2) * (kTcRows * 128) + off, 16, 1024),
             sdesc_sw128(aK + (k >> 2) * (kTcMaxRows * 128) + off, 16, 1024), id_s, k > 0);
    }
    tc_commit(smem_u32(&bar_s));
  };
  const uint32_t id_o = idesc_bf16(kTcRows, 64, true);
  // O half hd = P V[:, 64 hd ..]; the V descriptor is formed once and
  // stepped by adding to its address field (16-byte units).
  auto issue_pv = [&](int hd, int NSt) {
    const uint64_t dv = sdesc_sw128(aV + hd * (kTcMaxRows * 128), kTcMaxRows * 128, 1024);
    const uint32_t dO = tm + kTcO;
    uint32_t aP = tm + kTcS;
    mma_ts_all(dO, aP, dv, id_o, false);
    mma_ts_all(dO, aP + 8, dv, id_o, true);
    for (int k = 1; k < NSt / 16; ++k) {  // K = keys, 16 a step (2048 bytes of V)
      aP += 16;
      const uint64_t bv = dv + (uint64_t)(k * 128);
      mma_ts_all(dO, aP, bv, id_o, true);
      mma_ts_all(dO, aP + 8, bv, id_o, true);
    }
    tc_commit(smem_u32(&bar_o));
  };
  bool ok = true;
  int ph_s = 0, ph_o = 0;
  auto wait_all = [&](uint64_t *bar, int &ph) {
    const bool got = mbar_wait(smem_u32(bar), (uint32_t)(ph & 1), abort);
    ph ^= 1;
    const bool all = __syncthreads_and(got) != 0;
    if (!all && tid == 0) {
      atomicOr(c.err, ERR_TIMEOUT);
      *abort = 1;
    }
    tc_fence_after();
    return all;
  };
  // The issuing thread waits for a tile's q rows before its S.
  auto wait_q = [&]() {  // thread 32
    const int q = s_q;
    const bool got = mbar_wait(smem_u32(&bar_q), (uint32_t)(q & 1), abort);
    if (got) {
      s_q = (q & 1) ^ 1;
    } else {
      atomicOr(c.err, ERR_TIMEOUT);
      *abort = 1;
    }
    return got;
  };
  // (K, written by the unit load, is visible to the tensor cores: the load
  // fenced the async proxy before its barrier.)
  if (tid == 32 && wait_q()) issue_s(0);
  for (int mt = 0; mt < n_mt && ok; ++mt) {
    // 1. S = Q K^T for the tile's keys is in tensor memory.
    if (!(ok = wait_all(&bar_s, ph_s))) break;
    if (tid == 32 && mt + 1 < n_mt) {  // S has read this tile's q rows
      load_q(mt + 1);
      s_q |= 2;
    }
    const int NSt = tile_cols(mt);
    const int half = ((NSt >> 1) + 15) & ~15;
    const int c_lo = upper ? half : 0, c_hi = upper ? NSt : half;
    const int nch = (c_hi - c_lo) >> 4;
    const int lim_w = lim_warp(mt, wq);  // warp-uniform: chunks from here on are all masked

    // 2. This thread's logits (at most kTcChunks 16-column chunks) read
    // from TMEM once, exponentiated against the thread's own maximum; the
    // row's maximum and sum come from an exchange with the partner warp.
    const bool valid = r < Jt * G && mt * Jt + r / G < C;
    const int lim = valid ? n0 + mt * Jt + r / G + 1 : 0;  // keys the row may see
    float e[kTcChunks][16];
    float mx = -INFINITY;
#pragma unroll
    for (int k = 0; k < kTcChunks; ++k)
      if (k < nch && c_lo + 16 * k < lim_w) tmem_ld16f_nowait(trow + kTcS + c_lo + 16 * k, e[k]);
    tmem_wait_ld();
    const uint64_t scale2 = pk2(scale, scale);
#pragma unroll
    for (int k = 0; k < kTcChunks; ++k) {
      if (k < nch && c_lo + 16 * k < lim_w) {
        if (c_lo + 16 * k + 16 <= lim) {  // the whole chunk is visible
#pragma unroll
          for (int j = 0; j < 16; j += 2) {
            upk2(mul2(pk2(e[k][j], e[k][j + 1]), scale2), e[k][j], e[k][j + 1]);
            mx = fmaxf(mx, fmaxf(e[k][j], e[k][j + 1]));
          }
        } else {
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const bool in = c_lo + 16 * k + j < lim;
            e[k][j] = in ? e[k][j] * scale : -INFINITY;
            mx = fmaxf(mx, e[k][j]);
          }
        }
      }
    }
    const float ref = mx == -INFINITY ? 0.f : mx;
    const uint64_t nref2 = pk2(-ref, -ref);
    uint64_t sm2 = pk2(0.f, 0.f);  // even and odd terms
#pragma unroll
    for (int k = 0; k < kTcChunks; ++k) {
      if (k < nch && c_lo + 16 * k < lim_w) {
#pragma unroll
        for (int j = 0; j < 16; j += 2) {
          float d0, d1;
          upk2(add2(pk2(e[k][j], e[k][j + 1]), nref2), d0, d1);
          e[k][j] = ex2(d0);  // exp2(-inf) = 0 for masked keys
          e[k][j + 1] = ex2(d1);
          sm2 = add2(sm2, pk2(e[k][j], e[k][j + 1]));
        }
      }
    }
    float sm;
    {
      float s0, s1;
      upk2(sm2, s0, s1);
      sm = s0 + s1;
    }
    // Warps w and w + 4 (the same 32 rows) exchange (max, sum) through
    // shared memory on a named barrier of their own; both merge the two
    // pairs in the same order, so they agree to the bit.
    const uint32_t bar_id = 1 + wq;
    (upper ? s_mh : s_ml)[r] = make_float2(mx, sm);
    asm volatile("bar.sync %0, 64;" ::"r"(bar_id) : "memory");
    const float2 lo2 = s_ml[r], hi2 = s_mh[r];
    const float M = fmaxf(lo2.x, hi2.x);
    const float L = (lo2.x == -INFINITY ? 0.f : lo2.y * ex2(lo2.x - M)) +
                    (hi2.x == -INFINITY ? 0.f : hi2.y * ex2(hi2.x - M));
    if (valid && !upper && !(L >= 1.f && L < INFINITY)) atomicOr(c.err, ERR_NONFINITE);
    // p = e * exp2(own max - row max) / row sum; rows past the tile's
    // queries have f = 0 and finite e, so exact zeros.
    const float f = valid && L > 0.f && mx > -INFINITY ? ex2(mx - M) / L : 0.f;
    const uint64_t f2 = pk2(f, f);
#pragma unroll
    for (int k = 0; k < kTcChunks; ++k) {
      if (k >= nch) continue;
      const uint32_t cp = trow + kTcS + c_lo + 16 * k;
      uint32_t hi[8], lo[8];
      if (c_lo + 16 * k < lim_w) {
#pragma unroll
        for (int j = 0; j < 16; j += 2) {
          const uint64_t p2 = mul2(pk2(e[k][j], e[k][j + 1]), f2);
          float p0, p1;
          upk2(p2, p0, p1);
          e[k][j] = p0;
          e[k][j + 1] = p1;
          const __nv_bfloat162 b = __floats2bfloat162_rn(p0, p1);
          hi[j >> 1] = *reinterpret_cast<const uint32_t *>(&b);
          float r0, r1;  // p - bf16(p), both terms at once
          upk2(add2(p2, pk2(-__low2float(b), -__high2float(b))), r0, r1);
          lo[j >> 1] = pack_bf16(r0, r1);
        }
        // P in place of the chunk's logits: 8 hi then 8 lo columns.
        tmem_st8(cp, hi);
        tmem_st8(cp + 8, lo);
        // The chunk's column sums over the warp's 32 rows, one slot per
        // lane quarter (summed in a fixed order below).
        int col;
        const float cs = colsum32(e[k], lane, col);
        if ((lane & 1) == 0) PART[wq * kTcMaxRows + c_lo + 16 * k + col] = cs;
      } else {  // every row of the warp is masked here: P = 0
#pragma unroll
        for (int j = 0; j < 8; ++j) hi[j] = 0u;
        tmem_st8(cp, hi);
        tmem_st8(cp + 8, hi);
      }
    }
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
    tc_fence_before();
    __syncthreads();
    tc_fence_after();

    // 3. O = P V, one 64-column half of the head dimension at a time:
    // P (hi and lo) from tensor memory, V MN-major from shared memory.
    if (tid == 0) issue_pv(0, NSt);
    // The scores: each key's column sums from the lane quarters whose
    // chunk held it, in a fixed order (warps 2 and up: warp 0 issues).
    if (const int key = tid - 64; key >= 0 && key < NSt && key < n) {
      float sc = 0.f;
#pragma unroll
      for (int q4 = 0; q4 < 4; ++q4)
        if ((key & ~15) < lim_warp(mt, q4)) sc += PART[q4 * kTcMaxRows + key];
      ACC[key] += sc * inv_g;
    }
    constexpr int osz = kOutBf16 ? 2 : 4;
    unsigned char *orow = nullptr;
    if (valid) {
      const int rq = r / G, tok = mt * Jt + rq, rg = r - rq * G;
      orow = reinterpret_cast<unsigned char *>(p.out) +
             ((((u.row0 + tok) * c.H + h) * G + rg) * 128) * osz;
    }
    for (int hd = 0; hd < 2 && ok; ++hd) {
      if (!(ok = wait_all(&bar_o, ph_o))) break;
      // After the second half, P has been read: the next tile's S may
      // overwrite it while this O half drains.
      if (hd == 1 && tid == 32 && mt + 1 < n_mt && wait_q()) issue_s(mt + 1);
      // This thread's row, 32 of the half's columns.
      float ov[2][16];
      const int c0 = (upper ? 32 : 0);
      tmem_ld16f_nowait(trow + kTcO + c0, ov[0]);
      tmem_ld16f_nowait(trow + kTcO + c0 + 16, ov[1]);
      tmem_wait_ld();
      // The second half's MMAs overwrite O once every thread has read the
      // first.  (After the second half, the next writer of O is the next
      // tile's first half, issued after that tile's fenced barrier.)
      if (hd == 0) {
        tc_fence_before();
        __syncthreads();
        tc_fence_after();
        if (tid == 0) issue_pv(1, NSt);
      }
      if (valid) {
#pragma unroll
        for (int k = 0; k < 2; ++k) {
          const int d0 = 64 * hd + c0 + 16 * k;
          if (kOutBf16) {
            uint32_t w[8];
#pragma unroll
            for (int jj = 0; jj < 8; ++jj) w[jj] = pack_bf16(ov[k][2 * jj], ov[k][2 * jj + 1]);
            reinterpret_cast<int4 *>(orow + d0 * 2)[0] = make_int4(w[0], w[1], w[2], w[3]);
            reinterpret_cast<int4 *>(orow + d0 * 2)[1] = make_int4(w[4], w[5], w[6], w[7]);
          } else {
#pragma unroll
            for (int jj = 0; jj < 4; ++jj)
              reinterpret_cast<float4 *>(orow + d0 * 4)[jj] =
                  make_float4(ov[k][4 * jj], ov[k][4 * jj + 1], ov[k][4 * jj + 2],
                              ov[k][4 * jj + 3]);
          }
        }
      }
    }
  }
  // After a timeout, wait (bounded) once more for tensor work in flight.
  // Only the barrier whose wait gave up has a commit outstanding (its phase
  // has the parity before the toggle); on the other, that parity names a
  // completed phase and the wait returns at once.
  if (!ok) {
    volatile int never = 0;
    if (tid == 32) {
      mbar_wait(smem_u32(&bar_s), (uint32_t)((ph_s ^ 1) & 1), &never);
      mbar_wait(smem_u32(&bar_o), (uint32_t)((ph_o ^ 1) & 1), &never);
      if (s_q & 2) mbar_wait(smem_u32(&bar_q), (uint32_t)(s_q & 1), &never);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tm, kTcCols);
  if (!ok) return;
  finish_unit<kTcMaxRows>(p, u, m, s_wsum);
}

}  // namespace

int absorb_max_chunk() { return kMaxChunk; }
int absorb_max_rows() { return kMaxRows; }

cudaError_t launch_absorb(const AbsorbParams &p, int kernel, const CUtensorMap *tmQ,
                          cudaStream_t st, int *ran) {
  if (p.chunk < 1 || p.chunk > kMaxChunk || p.c.G > 8 || p.c.d != 128 ||
      !p.c.kv_bf16)
    return cudaErrorInvalidValue;
  const int units = p.c.S * p.nl * p.c.H;
  // The tensor-memory kernel stages at most kTcMaxRows rows; larger units
  // (up to kMaxRows) take the mma.sync kernel.
  const bool tc = kernel != 1 && p.max_rows <= kTcMaxRows && tmQ;
  if (ran) *ran = tc ? 0 : 1;
  if (tc) {
    auto kern = p.c.out_bf16 ? absorb_tc_kernel<true> : absorb_tc_kernel<false>;
    cudaError_t e = cudaFuncSetAttribute(
        kern, cudaFuncAttributeMaxDynamicSharedMemorySize, TcSmem::alloc);
    if (e != cudaSuccess) return e;
    return launch_pdl(kern, dim3(units), dim3(kThreads), (size_t)TcSmem::alloc, st, p, *tmQ);
  }
  auto kern = p.c.out_bf16 ? absorb_kernel<true> : absorb_kernel<false>;
  cudaError_t e = cudaFuncSetAttribute(
      kern, cudaFuncAttributeMaxDynamicSharedMemorySize, AbsorbSmem::bytes);
  if (e != cudaSuccess) return e;
  return launch_pdl(kern, dim3(units), dim3(kThreads), (size_t)AbsorbSmem::bytes, st, p);
}

}  // namespace kvr
