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

// A float's order as an unsigned integer, negative values included.
__device__ __forceinline__ unsigned ord_bits(float z) {
  const unsigned b = __float_as_uint(z);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// Higher z first, then lower position.
__device__ __forceinline__ unsigned long long rkv_key(float z, int32_t p) {
  return (static_cast<unsigned long long>(ord_bits(z)) << 32) |
         static_cast<unsigned long long>(0xFFFFFFFFu - static_cast<unsigned>(p));
}

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
  if (tid == 0) c.state[4 * x.u] = nk;
}

template <typename T, int D>
cudaError_t rkv_dispatch(const CacheView &c, int lb, int nl, int max_rows,
                         int B, int W, float lam, cudaStream_t st) {
  const int nk = B + W;
  const int max_list = max(1, min(nk, max_rows - nk));
  const size_t list_bytes = 2 * (size_t)max_list * sizeof(int);
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
