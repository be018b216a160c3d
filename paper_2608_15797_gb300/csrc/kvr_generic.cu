// kvr_generic.cu -- generic decode-step kernels of libkvr: one CTA per unit
// (sequence, layer, KV head), any head_dim in {64, 128}, G <= 8, fp32 or
// bf16 elements.  These serve every shape; the bf16 / d=128 steady state has
// a faster fused kernel (kvr_fused.cu).
//
// attend_score_kernel: Eq. 1 Attn(q_t, C) for the G query heads of one KV
//   head plus the accumulated-attention update of Sec. 2.1 (score += mean over
//   the G heads of the row's probability).  Logits live in shared memory when
//   they fit, else in the cache's per-unit logit scratch; K and V are each
//   read once.
// evict_kernel: TopB of Eq. 1 with the protected recent window of Sec. 4.1:
//   a block radix select of the B-th best (score, -position) key among the
//   non-window rows, then an in-place compaction that moves the survivors
//   lying beyond the new length into the freed slots below it.
#include <cuda_bf16.h>
#include <math.h>

#include "kvr_device.cuh"
#include "kvr_internal.h"

namespace kvr {
namespace {

using namespace dev;

struct Unit {
  int s, lr, l, h;
  size_t u;
};

__device__ __forceinline__ Unit unit_of(const CacheView &c, int lb, int nl) {
  Unit x;
  const int b = blockIdx.x;
  x.h = b % c.H;
  x.lr = (b / c.H) % nl;
  x.s = b / (c.H * nl);
  x.l = lb + x.lr;
  x.u = ((size_t)x.s * c.L + x.l) * c.H + x.h;
  return x;
}

// Dynamic shared memory of attend_score_kernel (floats).
__host__ __device__ constexpr int attend_fixed_floats(int D) {
  return kMaxG * D                           // q
         + (kThreads / (D / 2)) * kMaxG * D  // PV partials per row group
         + 2 * kMaxG;                        // max and 1/sum per head
}

// kExtScratch: logits always go to `ext`, one [G][max_rows] block per CTA,
// instead of shared memory or the cache's own scratch area.
template <typename T, typename O, int D, bool kExtScratch = false>
__global__ void __launch_bounds__(kThreads)
    attend_score_kernel(CacheView c, StepArgs a, int logits_in_smem,
                        float *ext) {
  pdl_begin();
  extern __shared__ float smem[];
  constexpr int P = D / 2;         // dimension pairs
  constexpr int R = kThreads / P;  // row groups of the PV pass
  constexpr int E = D / 32;        // elements per lane in the QK pass
  float *qs = smem;
  float *red = qs + kMaxG * D;
  float *stat_m = red + R * kMaxG * D;
  float *stat_iz = stat_m + kMaxG;
  float *lg_s = stat_iz + kMaxG;

  const int G = c.G;
  const Unit x = unit_of(c, a.lb, a.nl);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

  const int n0 = c.state[4 * x.u];
  if (n0 + 1 > c.cap) {
    if (tid == 0) atomicOr(c.err, ERR_CAPACITY);
    return;
  }
  const int n = n0 + 1;
  T *Ku = reinterpret_cast<T *>(c.K) + x.u * (size_t)c.cap * D;
  T *Vu = reinterpret_cast<T *>(c.V) + x.u * (size_t)c.cap * D;
  float *su = c.score + x.u * (size_t)c.sstride;
  int32_t *pu = c.pos + x.u * (size_t)c.sstride;
  const size_t kv_row =
      (((size_t)x.s * a.nl + x.lr) * a.chunk + a.tok) * c.H + x.h;
  const size_t q_row = kv_row * G;
  const T *qg = reinterpret_cast<const T *>(a.q) + q_row * D;
  const T *kn = reinterpret_cast<const T *>(a.k_new) + kv_row * D;
  const T *vn = reinterpret_cast<const T *>(a.v_new) + kv_row * D;

  // Append: the new row goes to slot n0 with score 0 and the next position.
  for (int i = tid; i < G * D; i += kThreads) qs[i] = to_f(qg[i]);
  for (int i = tid; i < D; i += kThreads) {
    Ku[(size_t)n0 * D + i] = kn[i];
    Vu[(size_t)n0 * D + i] = vn[i];
  }
  const int newest = c.state[4 * x.u + 1];
  if (tid == 0) {
    pu[n0] = newest;
    su[n0] = 0.f;
  }
  __syncthreads();

  float *lg = kExtScratch ? ext + (size_t)blockIdx.x * G * a.max_rows
              : logits_in_smem ? lg_s
                               : c.logits + x.u * (size_t)G * c.cap;
  const int ls = (kExtScratch || logits_in_smem) ? a.max_rows : c.cap;

  // Logits l_{g,i} = scale * <q_g, k_i>: one warp per row.
  for (int i = warp; i < n; i += kWarps) {
    const T *kr = Ku + (size_t)i * D + lane * E;
    float kv[E];
#pragma unroll
    for (int e = 0; e < E; e += 2) {
      float2 t = ld2(kr + e);
      kv[e] = t.x;
      kv[e + 1] = t.y;
    }
#pragma unroll
    for (int g = 0; g < kMaxG; ++g) {
      if (g < G) {
        float acc = 0.f;
#pragma unroll
        for (int e = 0; e < E; ++e) acc += qs[g * D + lane * E + e] * kv[e];
        acc = warp_sum(acc);
        if (lane == 0) lg[(size_t)g * ls + i] = acc * c.scale;
      }
    }
  }
  __syncthreads();

  // Softmax statistics: warp g owns query head g.
  if (warp < G) {
    const float *lr = lg + (size_t)warp * ls;
    float m = -INFINITY;
    for (int i = lane; i < n; i += 32) m = fmaxf(m, lr[i]);
    m = warp_max(m);
    float z = 0.f;
    for (int i = lane; i < n; i += 32) z += expf(lr[i] - m);
    z = warp_sum(z);
    if (lane == 0) {
      stat_m[warp] = m;
      stat_iz[warp] = 1.f / z;
      if (!(z >= 1.f) || !isfinite(z) || !isfinite(m)) atomicOr(c.err, ERR_NONFINITE);
    }
  }
  __syncthreads();

  // Probabilities, and the accumulated-attention update with their mean.
  const float inv_g = 1.f / (float)G;
  for (int i = tid; i < n; i += kThreads) {
    float acc = 0.f;
    for (int g = 0; g < G; ++g) {
      const float p = expf(lg[(size_t)g * ls + i] - stat_m[g]) * stat_iz[g];
      lg[(size_t)g * ls + i] = p;
      acc += p;
    }
    su[i] += acc * inv_g;
  }
  __syncthreads();

  // out_g = sum_i p_{g,i} v_i: thread (row group, dimension pair).
  const int dp = tid % P, rg = tid / P;
  float acc[kMaxG][2];
#pragma unroll
  for (int g = 0; g < kMaxG; ++g) acc[g][0] = acc[g][1] = 0.f;
  for (int i = rg; i < n; i += R) {
    const float2 v = ld2(Vu + (size_t)i * D + 2 * dp);
#pragma unroll
    for (int g = 0; g < kMaxG; ++g) {
      if (g < G) {
        const float p = lg[(size_t)g * ls + i];
        acc[g][0] += p * v.x;
        acc[g][1] += p * v.y;
      }
    }
  }
#pragma unroll
  for (int g = 0; g < kMaxG; ++g) {
    red[(rg * kMaxG + g) * D + 2 * dp] = acc[g][0];
    red[(rg * kMaxG + g) * D + 2 * dp + 1] = acc[g][1];
  }
  __syncthreads();
  O *og = reinterpret_cast<O *>(a.out) + q_row * D;
  for (int i = tid; i < G * D; i += kThreads) {
    const int g = i / D, dd = i % D;
    float o = 0.f;
#pragma unroll
    for (int r = 0; r < R; ++r) o += red[(r * kMaxG + g) * D + dd];
    st1(og + i, o);
  }
  if (tid == 0) {
    c.state[4 * x.u] = n;
    c.state[4 * x.u + 1] = newest + 1;
    c.state[4 * x.u + 2] = 0;  // the R-KV key sum no longer matches
  }
}

template <typename T, int D>
__global__ void __launch_bounds__(kThreads)
    evict_kernel(CacheView c, int lb, int nl, int B, int W) {
  pdl_begin();
  __shared__ unsigned hist[256];
  __shared__ unsigned long long s_prefix;
  __shared__ int s_need, s_base, s_count;
  __shared__ int s_wsum[kWarps];
  extern __shared__ int lists[];  // holes | movers, each max_list entries

  const Unit x = unit_of(c, lb, nl);
  const int tid = threadIdx.x;
  const int n = c.state[4 * x.u];
  if (n <= B + W) return;
  T *Ku = reinterpret_cast<T *>(c.K) + x.u * (size_t)c.cap * D;
  T *Vu = reinterpret_cast<T *>(c.V) + x.u * (size_t)c.cap * D;
  float *su = c.score + x.u * (size_t)c.sstride;
  int32_t *pu = c.pos + x.u * (size_t)c.sstride;
  // The W most recent positions are protected; a row is a candidate iff its
  // position is at most newest - W.
  const int wlo = c.state[4 * x.u + 1] - 1 - W;

  // TopB: by rank when every row has its own thread, else by a radix
  // select of the B-th largest candidate key.
  __shared__ unsigned long long s_key[kThreads];
  __shared__ unsigned char s_keep[kThreads];
  const bool by_rank = n <= kThreads;
  unsigned long long thr = ~0ull;
  if (by_rank)
    block_rank_keep(
        n, B, [&](int i) { return pu[i] <= wlo; },
        [&](int i) { return rank_key(su[i], pu[i]); }, s_key, s_keep);
  else if (B > 0)
    thr = block_select(
        n, B, [&](int i) { return pu[i] <= wlo; },
        [&](int i) { return rank_key(su[i], pu[i]); }, hist, &s_prefix,
        &s_need);
  auto keep = [&](int i) {
    if (by_rank) return s_keep[i] != 0;
    const int32_t p = pu[i];
    return p > wlo || (B > 0 && rank_key(su[i], p) >= thr);
  };

  // New length = number of kept rows (B + W whenever the window is intact).
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
  // Move every survivor beyond nk into a freed slot below it (disjoint).
  const int lane = tid & 31, warp = tid >> 5;
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
      su[dst] = su[src];
      pu[dst] = pu[src];
    }
  }
  if (tid == 0) {
    c.state[4 * x.u] = nk;
    c.state[4 * x.u + 2] = 0;  // the R-KV key sum no longer matches
  }
}

// Copy one sequence's prompt rows [L][H][n][d] into its slabs.
template <typename T, int D>
__global__ void load_kernel(CacheView c, int seq, const T *k, const T *v,
                            int n, int first_pos) {
  const int lh = blockIdx.x;  // layer * H + head
  const size_t u = (size_t)seq * c.L * c.H + lh;
  const int r0 = blockIdx.y * 32;
  const int r1 = min(r0 + 32, n);
  T *Ku = reinterpret_cast<T *>(c.K) + u * (size_t)c.cap * D;
  T *Vu = reinterpret_cast<T *>(c.V) + u * (size_t)c.cap * D;
  const T *ks = k + (size_t)lh * n * D;
  const T *vs = v + (size_t)lh * n * D;
  constexpr int kChunks = D * (int)sizeof(T) / 16;
  for (int q = threadIdx.x; q < (r1 - r0) * kChunks; q += blockDim.x) {
    const size_t r = r0 + q / kChunks, cidx = q % kChunks;
    reinterpret_cast<int4 *>(Ku + r * D)[cidx] =
        reinterpret_cast<const int4 *>(ks + r * D)[cidx];
    reinterpret_cast<int4 *>(Vu + r * D)[cidx] =
        reinterpret_cast<const int4 *>(vs + r * D)[cidx];
  }
  for (int r = r0 + threadIdx.x; r < r1; r += blockDim.x) {
    c.score[u * c.sstride + r] = 0.f;
    c.pos[u * c.sstride + r] = first_pos + r;
  }
  if (blockIdx.y == 0 && threadIdx.x == 0) {
    c.state[4 * u] = n;
    c.state[4 * u + 1] = first_pos + n;
    c.state[4 * u + 2] = 0;  // no R-KV key sum yet
  }
}

template <typename T, typename O, int D>
cudaError_t attend_dispatch(const CacheView &c, const StepArgs &a,
                            cudaStream_t st) {
  const size_t fixed = attend_fixed_floats(D) * sizeof(float);
  const size_t lg = (size_t)kMaxG * a.max_rows * sizeof(float);
  int dev = 0, optin = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  const int in_smem = fixed + lg <= (size_t)optin ? 1 : 0;
  const size_t bytes = fixed + (in_smem ? lg : 0);
  auto kern = attend_score_kernel<T, O, D>;
  cudaError_t e = cudaFuncSetAttribute(
      kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  if (e != cudaSuccess) return e;
  const int grid = c.S * a.nl * c.H;
  return launch_pdl(kern, dim3(grid), dim3(kThreads), bytes, st, c, a, in_smem,
                    static_cast<float *>(nullptr));
}

template <typename T, typename O, int D>
cudaError_t attend_ext_dispatch(const CacheView &c, const StepArgs &a,
                                float *ext, cudaStream_t st) {
  const size_t bytes = attend_fixed_floats(D) * sizeof(float);
  auto kern = attend_score_kernel<T, O, D, true>;
  cudaError_t e = cudaFuncSetAttribute(
      kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  if (e != cudaSuccess) return e;
  return launch_pdl(kern, dim3(c.S * a.nl * c.H), dim3(kThreads), bytes, st, c,
                    a, 0, ext);
}

template <typename T, int D>
cudaError_t evict_dispatch(const CacheView &c, int lb, int nl, int max_rows,
                           int B, int W, cudaStream_t st) {
  const int nk = B + W;
  const int max_list = max(1, min(nk, max_rows - nk));
  const size_t bytes = 2 * (size_t)max_list * sizeof(int);
  auto kern = evict_kernel<T, D>;
  cudaError_t e = cudaFuncSetAttribute(
      kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  if (e != cudaSuccess) return e;
  return launch_pdl(kern, dim3(c.S * nl * c.H), dim3(kThreads), bytes, st, c,
                    lb, nl, B, W);
}

}  // namespace

cudaError_t launch_attend_score_generic(const CacheView &c, const StepArgs &a,
                                        cudaStream_t st) {
  if (c.kv_bf16) {
    if (c.d == 128)
      return c.out_bf16
                 ? attend_dispatch<__nv_bfloat16, __nv_bfloat16, 128>(c, a, st)
                 : attend_dispatch<__nv_bfloat16, float, 128>(c, a, st);
    return c.out_bf16
               ? attend_dispatch<__nv_bfloat16, __nv_bfloat16, 64>(c, a, st)
               : attend_dispatch<__nv_bfloat16, float, 64>(c, a, st);
  }
  if (c.d == 128)
    return c.out_bf16 ? attend_dispatch<float, __nv_bfloat16, 128>(c, a, st)
                      : attend_dispatch<float, float, 128>(c, a, st);
  return c.out_bf16 ? attend_dispatch<float, __nv_bfloat16, 64>(c, a, st)
                    : attend_dispatch<float, float, 64>(c, a, st);
}

cudaError_t launch_attend_score_ext_scratch(const CacheView &c,
                                            const StepArgs &a, float *ext,
                                            cudaStream_t st) {
  if (c.kv_bf16) {
    if (c.d == 128)
      return c.out_bf16 ? attend_ext_dispatch<__nv_bfloat16, __nv_bfloat16,
                                              128>(c, a, ext, st)
                        : attend_ext_dispatch<__nv_bfloat16, float, 128>(
                              c, a, ext, st);
    return c.out_bf16
               ? attend_ext_dispatch<__nv_bfloat16, __nv_bfloat16, 64>(c, a,
                                                                        ext, st)
               : attend_ext_dispatch<__nv_bfloat16, float, 64>(c, a, ext, st);
  }
  if (c.d == 128)
    return c.out_bf16
               ? attend_ext_dispatch<float, __nv_bfloat16, 128>(c, a, ext, st)
               : attend_ext_dispatch<float, float, 128>(c, a, ext, st);
  return c.out_bf16 ? attend_ext_dispatch<float, __nv_bfloat16, 64>(c, a, ext, st)
                    : attend_ext_dispatch<float, float, 64>(c, a, ext, st);
}

cudaError_t launch_evict_generic(const CacheView &c, int lb, int nl,
                                 int max_rows, int budget, int window,
                                 cudaStream_t st) {
  if (c.kv_bf16)
    return c.d == 128 ? evict_dispatch<__nv_bfloat16, 128>(c, lb, nl, max_rows,
                                                           budget, window, st)
                      : evict_dispatch<__nv_bfloat16, 64>(c, lb, nl, max_rows,
                                                          budget, window, st);
  return c.d == 128
             ? evict_dispatch<float, 128>(c, lb, nl, max_rows, budget, window, st)
             : evict_dispatch<float, 64>(c, lb, nl, max_rows, budget, window, st);
}

cudaError_t launch_load(const CacheView &c, int seq, const void *k,
                        const void *v, int n_rows, int first_pos,
                        cudaStream_t st) {
  // At least one row-block so that an empty prompt still resets the length.
  dim3 grid(c.L * c.H, n_rows > 0 ? (n_rows + 31) / 32 : 1);
  if (c.kv_bf16) {
    if (c.d == 128)
      load_kernel<__nv_bfloat16, 128><<<grid, 256, 0, st>>>(
          c, seq, (const __nv_bfloat16 *)k, (const __nv_bfloat16 *)v, n_rows,
          first_pos);
    else
      load_kernel<__nv_bfloat16, 64><<<grid, 256, 0, st>>>(
          c, seq, (const __nv_bfloat16 *)k, (const __nv_bfloat16 *)v, n_rows,
          first_pos);
  } else {
    if (c.d == 128)
      load_kernel<float, 128><<<grid, 256, 0, st>>>(
          c, seq, (const float *)k, (const float *)v, n_rows, first_pos);
    else
      load_kernel<float, 64><<<grid, 256, 0, st>>>(
          c, seq, (const float *)k, (const float *)v, n_rows, first_pos);
  }
  return cudaGetLastError();
}

cudaError_t launch_init(const CacheView &c, cudaStream_t st) {
  const size_t units = (size_t)c.S * c.L * c.H;
  cudaError_t e = cudaMemsetAsync(c.state, 0, units * 4 * sizeof(int32_t), st);
  if (e == cudaSuccess) e = cudaMemsetAsync(c.err, 0, 16, st);
  return e;
}

}  // namespace kvr
