// kvr_rkv.cu -- eviction with the redundancy-aware score of R-KV, the policy
// the paper's base model uses (App. C: cached tokens are scored by a mix of
// query-attention importance and key redundancy by cosine similarity, with
// mix weight lambda; the top B plus a recent window are kept).  The paper
// prints no formula; the library's reading, for a unit with n live rows,
// window rows (the W most recent) and candidates C (the rest):
//   r_i = (1 / (n - 1)) sum over live j != i of cos(k_i, k_j)
//   R_i = softmax over C of r,   I_i = s_i / sum over C of s
//   z_i = lambda I_i - (1 - lambda) R_i
// and the B candidates first by (z descending, position ascending) stay.
//
// The mean cosine needs no n x n similarity matrix: with khat the
// normalised keys, sum over j of cos(k_i, k_j) = khat_i . (sum over j of
// khat_j).  One CTA per unit therefore makes two passes over its keys (the
// first sums the normalised keys, the second takes each candidate's dot with
// that sum), reduces the softmax and importance normalisers, and then selects
// and compacts like the accumulated-attention eviction (block radix select
// on (z, position), survivors above the new length moved into freed slots).
// Units of at most 128 rows (the steady state) take one warp each (below).
// A unit of at most 256 rows whose keys fit in 96 KB is first staged in
// shared memory (keys, scores, positions and z), with 16-byte loads; each
// lane then reads a contiguous slice of every key.  Longer units read their
// keys from global memory and keep z in the unit's logit scratch.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "kvr_device.cuh"
#include "kvr_internal.h"

namespace kvr {
namespace {

using namespace dev;

// Packed fp32 pairs (round to nearest, no flush).
__device__ __forceinline__ uint64_t pk2(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void upk2(uint64_t v, float &lo, float &hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t fma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}

using dev::ord_bits;
using dev::rkv_key;

// The unit of this CTA: blocks run over (sequence, layer in [lb, lb + nl),
// KV head), head fastest.
__device__ __forceinline__ size_t unit_index(const CacheView &c, int lb,
                                             int nl) {
  const int b = blockIdx.x;
  const int h = b % c.H, lr = (b / c.H) % nl, s = b / (c.H * nl);
  return ((size_t)s * c.L + lb + lr) * c.H + h;
}

template <typename Op>
__device__ float block_reduce(float v, Op op, float *s_red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = op(v, __shfl_xor_sync(0xffffffffu, v, o));
  if (lane == 0) s_red[warp] = v;
  __syncthreads();
  float r = s_red[0];
  for (int w = 1; w < kWarps; ++w) r = op(r, s_red[w]);
  __syncthreads();
  return r;
}

constexpr int kStageRows = kThreads;
constexpr size_t kStageKeyBytes = 96 * 1024;

template <typename T, int D>
constexpr bool stageable() {
  return (size_t)kStageRows * D * sizeof(T) <= kStageKeyBytes;
}

// Shared-memory layout of a staged unit of up to `rows` rows (a multiple of
// 4): keys [rows][D], then z, scores and positions [rows], then the
// holes | movers lists.
template <typename T, int D>
struct Staged {
  size_t keys, z, score, pos, lists;
  __host__ __device__ explicit Staged(int rows)
      : keys(0),
        z((size_t)rows * D * sizeof(T)),
        score(z + (size_t)rows * sizeof(float)),
        pos(score + (size_t)rows * sizeof(float)),
        lists(pos + (size_t)rows * sizeof(int32_t)) {}
};

template <typename T, int D, bool kStaged>
__global__ void __launch_bounds__(kThreads)
    rkv_evict_kernel(CacheView c, int lb, int nl, int B, int W, float lam,
                     int srows) {
  pdl_begin();
  constexpr int kPer = D / 32;  // key elements per lane: a contiguous slice
  __shared__ unsigned hist[256];
  __shared__ unsigned long long s_prefix;
  __shared__ int s_need, s_base, s_count;
  __shared__ int s_wsum[kWarps];
  __shared__ float s_red[kWarps];
  __shared__ float s_S[kWarps][D];
  extern __shared__ __align__(16) unsigned char dyn[];

  const struct { size_t u; } x = {unit_index(c, lb, nl)};
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int n = c.state[4 * x.u];
  if (n <= B + W) return;
  T *Ku = reinterpret_cast<T *>(c.K) + x.u * (size_t)c.cap * D;
  T *Vu = reinterpret_cast<T *>(c.V) + x.u * (size_t)c.cap * D;
  float *su_g = c.score + x.u * (size_t)c.sstride;
  int32_t *pu_g = c.pos + x.u * (size_t)c.sstride;
  const int wlo = c.state[4 * x.u + 1] - 1 - W;
  // Where the pass reads keys, scores, positions and z.
  const T *Kr = Ku;
  float *su = su_g, *z = c.logits + x.u * (size_t)c.G * c.cap;
  int32_t *pu = pu_g;
  int *lists = reinterpret_cast<int *>(dyn);
  if constexpr (kStaged) {
    const Staged<T, D> L(srows);
    T *ks = reinterpret_cast<T *>(dyn + L.keys);
    const int n16 = n * D * (int)sizeof(T) / 16;
    for (int q = tid; q < n16; q += kThreads)
      reinterpret_cast<int4 *>(ks)[q] = reinterpret_cast<const int4 *>(Ku)[q];
    su = reinterpret_cast<float *>(dyn + L.score);
    pu = reinterpret_cast<int32_t *>(dyn + L.pos);
    z = reinterpret_cast<float *>(dyn + L.z);
    for (int i = tid; i < n; i += kThreads) {
      su[i] = su_g[i];
      pu[i] = pu_g[i];
    }
    lists = reinterpret_cast<int *>(dyn + L.lists);
    Kr = ks;
    __syncthreads();
  }

  // Pass 1: S = sum of the normalised keys of every live row (warp per row).
  float acc[kPer];
#pragma unroll
  for (int j = 0; j < kPer; ++j) acc[j] = 0.f;
  for (int i = warp; i < n; i += kWarps) {
    const T *kr = Kr + (size_t)i * D + lane * kPer;
    float v[kPer], ss = 0.f;
#pragma unroll
    for (int j = 0; j < kPer; ++j) {
      v[j] = to_f(kr[j]);
      ss = fmaf(v[j], v[j], ss);
    }
    ss = warp_sum(ss);
    const float inv = ss > 0.f ? 1.f / sqrtf(ss) : 0.f;
#pragma unroll
    for (int j = 0; j < kPer; ++j) acc[j] = fmaf(v[j], inv, acc[j]);
  }
#pragma unroll
  for (int j = 0; j < kPer; ++j) s_S[warp][lane * kPer + j] = acc[j];
  __syncthreads();
  for (int dd = tid; dd < D; dd += kThreads) {
    float t = 0.f;
    for (int w = 0; w < kWarps; ++w) t += s_S[w][dd];
    s_S[0][dd] = t;
  }
  __syncthreads();

  // Pass 2: each candidate's mean cosine with the other live rows.
  const float inv_n1 = 1.f / static_cast<float>(n - 1);
  for (int i = warp; i < n; i += kWarps) {
    if (pu[i] > wlo) continue;  // window rows are not ranked
    const T *kr = Kr + (size_t)i * D + lane * kPer;
    float ss = 0.f, dot = 0.f;
#pragma unroll
    for (int j = 0; j < kPer; ++j) {
      const float v = to_f(kr[j]);
      ss = fmaf(v, v, ss);
      dot = fmaf(v, s_S[0][lane * kPer + j], dot);
    }
    ss = warp_sum(ss);
    dot = warp_sum(dot);
    const float inv = ss > 0.f ? 1.f / sqrtf(ss) : 0.f;
    const float self = ss > 0.f ? 1.f : 0.f;  // cos(k_i, k_i)
    if (lane == 0) z[i] = (dot * inv - self) * inv_n1;
  }
  __syncthreads();

  // Normalisers over the candidates: max r, sum exp(r - max), sum s.
  float mr = -INFINITY, ssum = 0.f;
  for (int i = tid; i < n; i += kThreads)
    if (pu[i] <= wlo) {
      mr = fmaxf(mr, z[i]);
      ssum += su[i];
    }
  mr = block_reduce(mr, [](float a, float b) { return fmaxf(a, b); }, s_red);
  ssum = block_reduce(ssum, [](float a, float b) { return a + b; }, s_red);
  float esum = 0.f;
  for (int i = tid; i < n; i += kThreads)
    if (pu[i] <= wlo) esum += expf(z[i] - mr);
  esum = block_reduce(esum, [](float a, float b) { return a + b; }, s_red);
  const float inv_e = 1.f / esum;
  const float inv_s = ssum > 0.f ? 1.f / ssum : 0.f;
  for (int i = tid; i < n; i += kThreads)
    if (pu[i] <= wlo)
      z[i] = lam * (su[i] * inv_s) - (1.f - lam) * (expf(z[i] - mr) * inv_e);
  __syncthreads();

  // TopB on (z, position): by rank when every row has its own thread,
  // else by block radix select; then compaction as in the score eviction.
  __shared__ unsigned long long s_key[kThreads];
  __shared__ unsigned char s_keep[kThreads];
  const bool by_rank = n <= kThreads;
  unsigned long long thr = ~0ull;
  if (by_rank)
    block_rank_keep(
        n, B, [&](int i) { return pu[i] <= wlo; },
        [&](int i) { return rkv_key(z[i], pu[i]); }, s_key, s_keep);
  else if (B > 0)
    thr = block_select(
        n, B, [&](int i) { return pu[i] <= wlo; },
        [&](int i) { return rkv_key(z[i], pu[i]); }, hist, &s_prefix,
        &s_need);
  auto keep = [&](int i) {
    if (by_rank) return s_keep[i] != 0;
    const int32_t p = pu[i];
    return p > wlo || (B > 0 && rkv_key(z[i], p) >= thr);
  };
  if (tid == 0) s_count = 0;
  __syncthreads();
  int mine = 0;
  for (int i = tid; i < n; i += kThreads) mine += keep(i) ? 1 : 0;
  atomicAdd(&s_count, mine);
  __syncthreads();
  const int nk = s_count;
  if (nk != B + W) {
    if (tid == 0) atomicOr(c.err, ERR_LENGTH);
    return;
  }
  const int max_list = min(nk, n - nk);
  int *holes = lists, *movers = lists + max_list;
  const int nh = block_collect(0, nk, [&](int i) { return !keep(i); }, holes,
                               s_wsum, &s_base);
  const int nm = block_collect(nk, n, keep, movers, s_wsum, &s_base);
  if (nh != nm) {
    if (tid == 0) atomicOr(c.err, ERR_LENGTH);
    return;
  }
  constexpr int kChunks = D * (int)sizeof(T) / 16;
  for (int j = warp; j < nh; j += kWarps) {
    const int dst = holes[j], src = movers[j];
    const int4 *ks = reinterpret_cast<const int4 *>(Ku + (size_t)src * D);
    const int4 *vs = reinterpret_cast<const int4 *>(Vu + (size_t)src * D);
    int4 *kd = reinterpret_cast<int4 *>(Ku + (size_t)dst * D);
    int4 *vd = reinterpret_cast<int4 *>(Vu + (size_t)dst * D);
    for (int q = lane; q < kChunks; q += 32) {
      kd[q] = ks[q];
      vd[q] = vs[q];
    }
    if (lane == 0) {
      su_g[dst] = su[src];
      pu_g[dst] = pu[src];
    }
  }
  if (tid == 0) {
    c.state[4 * x.u] = nk;
    c.state[4 * x.u + 2] = 0;  // the kept key sum is the one-launch step's
  }
}

// ---- one warp per unit (units of at most 128 rows: the steady state) -------
//
// The same arithmetic with no CTA-wide synchronisation: eight units a CTA,
// one a warp.  In the key passes each half-warp takes one row (16 lanes x
// D/16 elements, 16-byte loads for bf16 d = 128), so a warp reads two rows a
// step and keeps D/16 elements of the normalised-key sum per lane; pass 1
// leaves each row's inverse norm in the row's scratch slot for pass 2.  For
// the selection every lane owns rows lane, lane + 32, ...; the e = (number
// of candidates) - B smallest keys are dropped by e warp-wide minimum
// searches (keys are unique: they end in the position), which is one search
// in the steady state, and ballots build the hole and mover lists.
constexpr int kWarpRows = 128;

template <typename T, int D>
__global__ void __launch_bounds__(kThreads)
    rkv_evict_warp_kernel(CacheView c, int lb, int nl, int B, int W, float lam,
                          int units) {
  pdl_begin();
  constexpr int kE = D / 16;  // elements of a row per half-warp lane
  constexpr int kR = kWarpRows / 32;
  __shared__ float s_r[kWarps][kWarpRows];
  __shared__ int s_list[kWarps][2][kWarpRows];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int ui = blockIdx.x * kWarps + warp;
  if (ui >= units) return;
  const int b = ui;
  const int hh = b % c.H, lr = (b / c.H) % nl, sq = b / (c.H * nl);
  const size_t u = ((size_t)sq * c.L + lb + lr) * c.H + hh;
  const int n = c.state[4 * u];
  if (n <= B + W) return;
  if (n > kWarpRows) {  // the host sized the launch from its mirror
    if (lane == 0) atomicOr(c.err, ERR_LENGTH);
    return;
  }
  T *Ku = reinterpret_cast<T *>(c.K) + u * (size_t)c.cap * D;
  T *Vu = reinterpret_cast<T *>(c.V) + u * (size_t)c.cap * D;
  float *su = c.score + u * (size_t)c.sstride;
  int32_t *pu = c.pos + u * (size_t)c.sstride;
  const int wlo = c.state[4 * u + 1] - 1 - W;
  const int half = lane >> 4, l16 = lane & 15;
  float *rs = s_r[warp];

  // kE elements of row i with vector loads (8, 16 or 32 bytes).
  auto load_row = [&](int i, float (&v)[kE]) {
    const T *kr = Ku + (size_t)i * D + l16 * kE;
    if constexpr (sizeof(T) == 2 && kE == 8) {
      const uint4 w = __ldg(reinterpret_cast<const uint4 *>(kr));
      const uint32_t x[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        v[2 * j] = __uint_as_float(x[j] << 16);
        v[2 * j + 1] = __uint_as_float(x[j] & 0xffff0000u);
      }
    } else if constexpr (sizeof(T) == 2 && kE == 4) {
      const uint2 w = __ldg(reinterpret_cast<const uint2 *>(kr));
      v[0] = __uint_as_float(w.x << 16);
      v[1] = __uint_as_float(w.x & 0xffff0000u);
      v[2] = __uint_as_float(w.y << 16);
      v[3] = __uint_as_float(w.y & 0xffff0000u);
    } else {
#pragma unroll
      for (int j = 0; j < kE; j += 4) {
        const float4 w = __ldg(reinterpret_cast<const float4 *>(kr + j));
        v[j] = w.x, v[j + 1] = w.y, v[j + 2] = w.z, v[j + 3] = w.w;
      }
    }
  };
  auto half_sum = [](float x) {
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
  };
  // Rows go kU pairs a step, all their loads issued before any is used.
  constexpr int kU = 5;
  auto load_rows = [&](int i0, float (&v)[kU][kE]) {
#pragma unroll
    for (int q = 0; q < kU; ++q) {
      const int i = i0 + 2 * q + half;
      if (i < n) load_row(i, v[q]);
      else {
#pragma unroll
        for (int j = 0; j < kE; ++j) v[q][j] = 0.f;
      }
    }
  };
  // Pass 1: S = sum of the normalised keys (this lane's kE dimensions, as
  // packed fp32 pairs); rs[i] = 1 / |k_i| (0 for a zero key).
  static_assert(kE % 2 == 0, "dimension pairs");
  uint64_t S2[kE / 2];
#pragma unroll
  for (int j = 0; j < kE / 2; ++j) S2[j] = pk2(0.f, 0.f);
  for (int i0 = 0; i0 < n; i0 += 2 * kU) {
    float v[kU][kE];
    load_rows(i0, v);
#pragma unroll
    for (int q = 0; q < kU; ++q) {
      uint64_t ss2 = pk2(0.f, 0.f);
#pragma unroll
      for (int j = 0; j < kE; j += 2) {
        const uint64_t x = pk2(v[q][j], v[q][j + 1]);
        ss2 = fma2(x, x, ss2);
      }
      float sa, sb;
      upk2(ss2, sa, sb);
      const float ss = half_sum(sa + sb);
      const float inv = ss > 0.f ? 1.f / sqrtf(ss) : 0.f;
      const uint64_t inv2 = pk2(inv, inv);
#pragma unroll
      for (int j = 0; j < kE; j += 2)
        S2[j / 2] = fma2(pk2(v[q][j], v[q][j + 1]), inv2, S2[j / 2]);
      const int i = i0 + 2 * q + half;
      if (l16 == 0 && i < n) rs[i] = inv;
    }
  }
#pragma unroll
  for (int j = 0; j < kE / 2; ++j) {
    float a, b;
    upk2(S2[j], a, b);
    a += __shfl_xor_sync(0xffffffffu, a, 16);
    b += __shfl_xor_sync(0xffffffffu, b, 16);
    S2[j] = pk2(a, b);
  }
  // Pass 2: each row's mean cosine with the other live rows (the lane that
  // wrote rs[i] in pass 1 reads and replaces it).
  const float inv_n1 = 1.f / (float)(n - 1);
  for (int i0 = 0; i0 < n; i0 += 2 * kU) {
    float v[kU][kE];
    load_rows(i0, v);
#pragma unroll
    for (int q = 0; q < kU; ++q) {
      const int i = i0 + 2 * q + half;
      uint64_t dot2 = pk2(0.f, 0.f);
#pragma unroll
      for (int j = 0; j < kE; j += 2)
        dot2 = fma2(pk2(v[q][j], v[q][j + 1]), S2[j / 2], dot2);
      float da, db;
      upk2(dot2, da, db);
      const float dot = half_sum(da + db);
      if (l16 == 0 && i < n) {
        const float inv = rs[i];
        rs[i] = (dot * inv - (inv > 0.f ? 1.f : 0.f)) * inv_n1;
      }
    }
  }
  __syncwarp();
  // This lane's rows: positions, scores, candidacy; normalisers over C.
  int ps[kR];
  float sc[kR], r[kR];
  bool cd[kR];
  float mr = -INFINITY, ssum = 0.f;
#pragma unroll
  for (int k = 0; k < kR; ++k) {
    const int i = lane + 32 * k;
    const bool in = i < n;
    ps[k] = in ? pu[i] : 0;
    sc[k] = in ? su[i] : 0.f;
    r[k] = in ? rs[i] : 0.f;
    cd[k] = in && ps[k] <= wlo;
    if (cd[k]) {
      mr = fmaxf(mr, r[k]);
      ssum += sc[k];
    }
  }
  mr = dev::warp_max(mr);
  ssum = dev::warp_sum(ssum);
  float esum = 0.f;
#pragma unroll
  for (int k = 0; k < kR; ++k)
    if (cd[k]) esum += expf(r[k] - mr);
  esum = dev::warp_sum(esum);
  const float inv_e = 1.f / esum, inv_s = ssum > 0.f ? 1.f / ssum : 0.f;
  unsigned long long key[kR];
  int ncand = 0;
#pragma unroll
  for (int k = 0; k < kR; ++k) {
    const float z = lam * (sc[k] * inv_s) - (1.f - lam) * (expf(r[k] - mr) * inv_e);
    key[k] = rkv_key(z, ps[k]);
    ncand += __popc(__ballot_sync(0xffffffffu, cd[k]));
  }
  // Drop the ncand - B smallest candidate keys, one warp-wide minimum at a
  // time; the rest of the candidates are the B largest.
  bool kp[kR], live[kR];
#pragma unroll
  for (int k = 0; k < kR; ++k) {
    kp[k] = lane + 32 * k < n;
    live[k] = cd[k];
  }
  for (int d = 0; d < ncand - B; ++d) {
    unsigned long long m = ~0ull;
#pragma unroll
    for (int k = 0; k < kR; ++k)
      if (live[k] && key[k] < m) m = key[k];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const unsigned long long x = __shfl_xor_sync(0xffffffffu, m, o);
      m = x < m ? x : m;
    }
#pragma unroll
    for (int k = 0; k < kR; ++k)
      if (live[k] && key[k] == m) live[k] = kp[k] = false;
  }
  int nk = 0;
#pragma unroll
  for (int k = 0; k < kR; ++k) nk += __popc(__ballot_sync(0xffffffffu, kp[k]));
  if (nk != B + W) {
    if (lane == 0) atomicOr(c.err, ERR_LENGTH);
    return;
  }
  // Holes (dropped rows below nk) and movers (kept rows at nk or above), in
  // row order; the j-th mover fills the j-th hole.
  int nh = 0, nm = 0;
#pragma unroll
  for (int k = 0; k < kR; ++k) {
    const int i = lane + 32 * k;
    const bool hole = i < nk && !kp[k];
    const bool mover = i >= nk && i < n && kp[k];
    const unsigned bh = __ballot_sync(0xffffffffu, hole);
    const unsigned bm = __ballot_sync(0xffffffffu, mover);
    const unsigned below = (1u << lane) - 1u;
    if (hole) s_list[warp][0][nh + __popc(bh & below)] = i;
    if (mover) s_list[warp][1][nm + __popc(bm & below)] = i;
    nh += __popc(bh);
    nm += __popc(bm);
  }
  __syncwarp();
  if (nh != nm) {
    if (lane == 0) atomicOr(c.err, ERR_LENGTH);
    return;
  }
  constexpr int kChunks = D * (int)sizeof(T) / 16;
  for (int j = 0; j < nh; ++j) {
    const int dst = s_list[warp][0][j], src = s_list[warp][1][j];
    const int4 *ks = reinterpret_cast<const int4 *>(Ku + (size_t)src * D);
    const int4 *vs = reinterpret_cast<const int4 *>(Vu + (size_t)src * D);
    int4 *kd = reinterpret_cast<int4 *>(Ku + (size_t)dst * D);
    int4 *vd = reinterpret_cast<int4 *>(Vu + (size_t)dst * D);
    for (int q = lane; q < kChunks; q += 32) {
      kd[q] = ks[q];
      vd[q] = vs[q];
    }
    if (lane == 0) {
      su[dst] = su[src];
      pu[dst] = pu[src];
    }
  }
  if (lane == 0) {
    c.state[4 * u] = nk;
    c.state[4 * u + 2] = 0;  // the kept key sum is the one-launch step's
  }
}

template <typename T, int D>
cudaError_t rkv_dispatch(const CacheView &c, int lb, int nl, int max_rows,
                         int B, int W, float lam, cudaStream_t st) {
  const int nk = B + W;
  const int max_list = max(1, min(nk, max_rows - nk));
  const size_t list_bytes = 2 * (size_t)max_list * sizeof(int);
  if (max_rows <= kWarpRows) {
    const int units = c.S * nl * c.H;
    return launch_pdl(rkv_evict_warp_kernel<T, D>,
                      dim3((units + kWarps - 1) / kWarps), dim3(kThreads), 0,
                      st, c, lb, nl, B, W, lam, units);
  }
  const bool staged = stageable<T, D>() && max_rows <= kStageRows;
  const int srows = (max_rows + 3) & ~3;
  const size_t bytes =
      staged ? Staged<T, D>(srows).lists + list_bytes : list_bytes;
  auto kern = staged ? rkv_evict_kernel<T, D, stageable<T, D>()>
                     : rkv_evict_kernel<T, D, false>;
  cudaError_t e = cudaFuncSetAttribute(
      kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  if (e != cudaSuccess) return e;
  return launch_pdl(kern, dim3(c.S * nl * c.H), dim3(kThreads), bytes, st, c,
                    lb, nl, B, W, lam, srows);
}

}  // namespace

cudaError_t launch_evict_rkv(const CacheView &c, int lb, int nl, int max_rows,
                             int budget, int window, float lam,
                             cudaStream_t st) {
  if (c.kv_bf16)
    return c.d == 128
               ? rkv_dispatch<__nv_bfloat16, 128>(c, lb, nl, max_rows, budget,
                                                  window, lam, st)
               : rkv_dispatch<__nv_bfloat16, 64>(c, lb, nl, max_rows, budget,
                                                 window, lam, st);
  return c.d == 128 ? rkv_dispatch<float, 128>(c, lb, nl, max_rows, budget,
                                               window, lam, st)
                    : rkv_dispatch<float, 64>(c, lb, nl, max_rows, budget,
                                              window, lam, st);
}

}  // namespace kvr
