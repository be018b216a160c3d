// kvr_fork.cu -- candidate kernels of libkvr (stepwise best-of-N, Sec. 2.2
// Eq. 2 and App. C): N candidates share the parent's live rows as a
// read-only prefix and keep private tails and private score copies.
//
// fork_attend_kernel: one CTA per (sequence, layer, KV head).  The prefix K
//   and V rows are staged in shared memory once and serve all N candidates;
//   each candidate then appends its row to its tail, computes Attn(q_t, C)
//   (Eq. 1) over prefix + tail for its G query heads, and adds the mean over
//   the heads of each row's probability to its own scores (Sec. 2.1).
// fork_commit_kernel: per unit, TopB with the protected window (Eq. 1,
//   Sec. 4.1) over the chosen candidate's prefix + tail rows and scores,
//   then the survivors are written into the parent: kept prefix rows below
//   the new length stay, every other survivor fills a freed parent slot.
#include <cuda_bf16.h>
#include <math.h>

#include <algorithm>

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

// Shared memory (bytes) of fork_attend_kernel before the staged prefix.
__host__ __device__ constexpr size_t fork_fixed_bytes(int D, int n_max) {
  return sizeof(float) * ((size_t)kMaxG * D                              // q
                          + (size_t)(kThreads / (D / 2)) * kMaxG * D      // PV
                          + 2 * kMaxG                                     // stats
                          + (size_t)kMaxG * n_max);                       // logits
}

template <typename T, typename O, int D>
__global__ void __launch_bounds__(kThreads)
    fork_attend_kernel(ForkView f, StepArgs a, int n_max) {
  pdl_begin();
  extern __shared__ __align__(16) unsigned char smem_raw[];
  constexpr int P = D / 2;         // dimension pairs
  constexpr int R = kThreads / P;  // row groups of the PV pass
  constexpr int E = D / 32;        // elements per lane in the QK pass
  const CacheView &c = f.p;
  const int G = c.G;
  float *qs = reinterpret_cast<float *>(smem_raw);
  float *red = qs + kMaxG * D;
  float *stat_m = red + R * kMaxG * D;
  float *stat_iz = stat_m + kMaxG;
  float *lg = stat_iz + kMaxG;  // [G][n_max]
  T *Ks = reinterpret_cast<T *>(smem_raw + fork_fixed_bytes(D, n_max));

  const Unit x = unit_of(c, a.lb, a.nl);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const size_t units = (size_t)c.S * c.L * c.H;
  const int np = c.state[4 * x.u];          // prefix rows
  const int base_pos = c.state[4 * x.u + 1];  // position of tail row 0
  T *Vs = Ks + (size_t)np * D;

  // Stage the prefix once for every candidate (16-byte vectors).
  {
    const int4 *kg = reinterpret_cast<const int4 *>(
        reinterpret_cast<const T *>(c.K) + x.u * (size_t)c.cap * D);
    const int4 *vg = reinterpret_cast<const int4 *>(
        reinterpret_cast<const T *>(c.V) + x.u * (size_t)c.cap * D);
    int4 *ks = reinterpret_cast<int4 *>(Ks), *vs = reinterpret_cast<int4 *>(Vs);
    const int chunks = np * D * (int)sizeof(T) / 16;
    for (int i = tid; i < chunks; i += kThreads) {
      ks[i] = kg[i];
      vs[i] = vg[i];
    }
  }

  for (int cand = 0; cand < f.N; ++cand) {
    const size_t cu = (size_t)cand * units + x.u;  // candidate's unit
    const int nt0 = f.tlen[cu];
    if (nt0 + 1 > f.tcap || np + nt0 + 1 > n_max) {
      if (tid == 0) atomicOr(c.err, ERR_CAPACITY);
      return;
    }
    T *Kt = reinterpret_cast<T *>(f.TK) + cu * (size_t)f.tcap * D;
    T *Vt = reinterpret_cast<T *>(f.TV) + cu * (size_t)f.tcap * D;
    float *ps = f.pscore + cu * (size_t)c.sstride;
    float *ts = f.tscore + cu * (size_t)f.tstride;
    const size_t kv_row =
        (((size_t)cand * c.S + x.s) * a.nl + x.lr) * c.H + x.h;
    const size_t q_row = kv_row * G;
    const T *qg = reinterpret_cast<const T *>(a.q) + q_row * D;
    const T *kn = reinterpret_cast<const T *>(a.k_new) + kv_row * D;
    const T *vn = reinterpret_cast<const T *>(a.v_new) + kv_row * D;

    // Append to the candidate's tail.
    for (int i = tid; i < G * D; i += kThreads) qs[i] = to_f(qg[i]);
    for (int i = tid; i < D; i += kThreads) {
      Kt[(size_t)nt0 * D + i] = kn[i];
      Vt[(size_t)nt0 * D + i] = vn[i];
    }
    if (tid == 0) {
      f.tpos[cu * f.tstride + nt0] = base_pos + nt0;
      ts[nt0] = 0.f;
    }
    __syncthreads();

    const int n = np + nt0 + 1;
    auto krow = [&](int i) -> const T * {
      return i < np ? Ks + (size_t)i * D : Kt + (size_t)(i - np) * D;
    };
    auto vrow = [&](int i) -> const T * {
      return i < np ? Vs + (size_t)i * D : Vt + (size_t)(i - np) * D;
    };

    // Logits: one warp per row.
    for (int i = warp; i < n; i += kWarps) {
      const T *kr = krow(i) + lane * E;
      float kv[E];
#pragma unroll
      for (int e = 0; e < E; e += 2) {
        const float2 t2 = ld2(kr + e);
        kv[e] = t2.x;
        kv[e + 1] = t2.y;
      }
#pragma unroll
      for (int g = 0; g < kMaxG; ++g) {
        if (g < G) {
          float acc = 0.f;
#pragma unroll
          for (int e = 0; e < E; ++e) acc += qs[g * D + lane * E + e] * kv[e];
          acc = warp_sum(acc);
          if (lane == 0) lg[(size_t)g * n_max + i] = acc * c.scale;
        }
      }
    }
    __syncthreads();

    if (warp < G) {
      const float *lr = lg + (size_t)warp * n_max;
      float m = -INFINITY;
      for (int i = lane; i < n; i += 32) m = fmaxf(m, lr[i]);
      m = warp_max(m);
      float z = 0.f;
      for (int i = lane; i < n; i += 32) z += expf(lr[i] - m);
      z = warp_sum(z);
      if (lane == 0) {
        stat_m[warp] = m;
        stat_iz[warp] = 1.f / z;
        if (!(z >= 1.f) || !isfinite(z) || !isfinite(m))
          atomicOr(c.err, ERR_NONFINITE);
      }
    }
    __syncthreads();

    // Probabilities and the candidate's accumulated-attention update.
    const float inv_g = 1.f / (float)G;
    for (int i = tid; i < n; i += kThreads) {
      float acc = 0.f;
      for (int g = 0; g < G; ++g) {
        const float p = expf(lg[(size_t)g * n_max + i] - stat_m[g]) * stat_iz[g];
        lg[(size_t)g * n_max + i] = p;
        acc += p;
      }
      if (i < np) ps[i] += acc * inv_g;
      else ts[i - np] += acc * inv_g;
    }
    __syncthreads();

    // out_g = sum_i p_{g,i} v_i.
    const int dp = tid % P, rg = tid / P;
    float acc[kMaxG][2];
#pragma unroll
    for (int g = 0; g < kMaxG; ++g) acc[g][0] = acc[g][1] = 0.f;
    for (int i = rg; i < n; i += R) {
      const float2 v = ld2(vrow(i) + 2 * dp);
#pragma unroll
      for (int g = 0; g < kMaxG; ++g) {
        if (g < G) {
          const float p = lg[(size_t)g * n_max + i];
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
    if (tid == 0) f.tlen[cu] = nt0 + 1;
    __syncthreads();  // shared buffers are reused by the next candidate
  }
}

template <typename T, int D>
__global__ void __launch_bounds__(kThreads)
    fork_commit_kernel(ForkView f, const int32_t *chosen, int B, int W) {
  pdl_begin();
  __shared__ unsigned hist[256];
  __shared__ unsigned long long s_prefix;
  __shared__ int s_need, s_base, s_count;
  __shared__ int s_wsum[kWarps];
  extern __shared__ int lists[];  // holes | movers
  const CacheView &c = f.p;
  const Unit x = unit_of(c, 0, c.L);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const size_t units = (size_t)c.S * c.L * c.H;
  const int cand = chosen[x.s];
  const size_t cu = (size_t)cand * units + x.u;
  const int np = c.state[4 * x.u], base_pos = c.state[4 * x.u + 1];
  const int nt = f.tlen[cu];
  const int n = np + nt;
  T *Ku = reinterpret_cast<T *>(c.K) + x.u * (size_t)c.cap * D;
  T *Vu = reinterpret_cast<T *>(c.V) + x.u * (size_t)c.cap * D;
  float *su = c.score + x.u * (size_t)c.sstride;
  int32_t *pu = c.pos + x.u * (size_t)c.sstride;
  const T *Kt = reinterpret_cast<const T *>(f.TK) + cu * (size_t)f.tcap * D;
  const T *Vt = reinterpret_cast<const T *>(f.TV) + cu * (size_t)f.tcap * D;
  const float *ps = f.pscore + cu * (size_t)c.sstride;
  const float *ts = f.tscore + cu * (size_t)f.tstride;
  const int32_t *tp = f.tpos + cu * (size_t)f.tstride;

  // Combined rows: r < np is parent slot r, r >= np is tail row r - np.
  auto score_of = [&](int r) { return r < np ? ps[r] : ts[r - np]; };
  auto pos_of = [&](int r) { return r < np ? pu[r] : tp[r - np]; };
  const int wlo = base_pos + nt - 1 - W;  // candidates: pos <= newest - W
  unsigned long long thr = 0;
  const bool evict = n > B + W;
  if (evict && B > 0)
    thr = block_select(
        n, B, [&](int r) { return pos_of(r) <= wlo; },
        [&](int r) { return rank_key(score_of(r), pos_of(r)); }, hist,
        &s_prefix, &s_need);
  auto keep = [&](int r) {
    if (!evict) return true;
    const int32_t pr = pos_of(r);
    return pr > wlo || (B > 0 && rank_key(score_of(r), pr) >= thr);
  };
  if (tid == 0) s_count = 0;
  __syncthreads();
  int mine = 0;
  for (int r = tid; r < n; r += kThreads) mine += keep(r) ? 1 : 0;
  atomicAdd(&s_count, mine);
  __syncthreads();
  const int nk = s_count;
  if (nk != (evict ? B + W : n)) {
    if (tid == 0) atomicOr(c.err, ERR_LENGTH);
    return;
  }
  // Staying rows: kept prefix rows below nk.  Holes: parent slots below nk
  // not staying.  Movers: every other kept row.  Disjoint sources and
  // destinations: moving prefix rows sit at or above nk.
  int *holes = lists, *movers = lists + nk;
  const int nh = block_collect(0, nk, [&](int j) { return j >= np || !keep(j); },
                               holes, s_wsum, &s_base);
  const int nm = block_collect(0, n, [&](int r) {
    return keep(r) && (r >= np || r >= nk);
  }, movers, s_wsum, &s_base);
  if (nh != nm) {
    if (tid == 0) atomicOr(c.err, ERR_LENGTH);
    return;
  }
  // The parent's scores become the candidate's for the staying rows.
  for (int j = tid; j < min(np, nk); j += kThreads)
    if (keep(j)) su[j] = ps[j];
  __syncthreads();
  constexpr int kChunks = D * (int)sizeof(T) / 16;
  for (int q = warp; q < nh; q += kWarps) {
    const int dst = holes[q], r = movers[q];
    const int4 *ks = reinterpret_cast<const int4 *>(
        r < np ? Ku + (size_t)r * D : Kt + (size_t)(r - np) * D);
    const int4 *vs = reinterpret_cast<const int4 *>(
        r < np ? Vu + (size_t)r * D : Vt + (size_t)(r - np) * D);
    int4 *kd = reinterpret_cast<int4 *>(Ku + (size_t)dst * D);
    int4 *vd = reinterpret_cast<int4 *>(Vu + (size_t)dst * D);
    for (int e = lane; e < kChunks; e += 32) {
      kd[e] = ks[e];
      vd[e] = vs[e];
    }
    if (lane == 0) {
      su[dst] = score_of(r);
      pu[dst] = pos_of(r);
    }
  }
  __syncthreads();
  if (tid == 0) {
    c.state[4 * x.u] = nk;
    c.state[4 * x.u + 1] = base_pos + nt;
    c.state[4 * x.u + 2] = 0;  // the R-KV key sum no longer matches
  }
}

template <typename T, typename O, int D>
cudaError_t fork_attend_dispatch(const ForkView &f, const StepArgs &a,
                                 int n_max, int max_prefix, cudaStream_t st) {
  const size_t bytes = fork_fixed_bytes(D, n_max) +
                       2 * (size_t)max_prefix * D * sizeof(T);
  auto kern = fork_attend_kernel<T, O, D>;
  cudaError_t e = cudaFuncSetAttribute(
      kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  if (e != cudaSuccess) return e;
  return launch_pdl(kern, dim3(f.p.S * a.nl * f.p.H), dim3(kThreads), bytes,
                    st, f, a, n_max);
}

template <typename T, int D>
cudaError_t fork_commit_dispatch(const ForkView &f, const int32_t *chosen,
                                 int max_rows, int B, int W, cudaStream_t st) {
  const size_t bytes = 2 * (size_t)std::max(1, max_rows) * sizeof(int);
  auto kern = fork_commit_kernel<T, D>;
  cudaError_t e = cudaFuncSetAttribute(
      kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  if (e != cudaSuccess) return e;
  return launch_pdl(kern, dim3(f.p.S * f.p.L * f.p.H), dim3(kThreads), bytes,
                    st, f, chosen, B, W);
}

}  // namespace

size_t fork_attend_smem_bytes(const CacheView &c, int n_max, int max_prefix) {
  const size_t e = c.kv_bf16 ? 2 : 4;
  return fork_fixed_bytes(c.d, n_max) + 2 * (size_t)max_prefix * c.d * e;
}

cudaError_t launch_fork_attend(const ForkView &f, const StepArgs &a, int n_max,
                               int max_prefix, cudaStream_t st) {
  const CacheView &c = f.p;
  if (c.kv_bf16) {
    if (c.d == 128)
      return c.out_bf16 ? fork_attend_dispatch<__nv_bfloat16, __nv_bfloat16, 128>(
                              f, a, n_max, max_prefix, st)
                        : fork_attend_dispatch<__nv_bfloat16, float, 128>(
                              f, a, n_max, max_prefix, st);
    return c.out_bf16 ? fork_attend_dispatch<__nv_bfloat16, __nv_bfloat16, 64>(
                            f, a, n_max, max_prefix, st)
                      : fork_attend_dispatch<__nv_bfloat16, float, 64>(
                            f, a, n_max, max_prefix, st);
  }
  if (c.d == 128)
    return c.out_bf16 ? fork_attend_dispatch<float, __nv_bfloat16, 128>(
                            f, a, n_max, max_prefix, st)
                      : fork_attend_dispatch<float, float, 128>(f, a, n_max,
                                                                max_prefix, st);
  return c.out_bf16 ? fork_attend_dispatch<float, __nv_bfloat16, 64>(
                          f, a, n_max, max_prefix, st)
                    : fork_attend_dispatch<float, float, 64>(f, a, n_max,
                                                             max_prefix, st);
}

cudaError_t launch_fork_commit(const ForkView &f, const int32_t *chosen,
                               int max_rows, int budget, int window,
                               cudaStream_t st) {
  const CacheView &c = f.p;
  if (c.kv_bf16)
    return c.d == 128 ? fork_commit_dispatch<__nv_bfloat16, 128>(
                            f, chosen, max_rows, budget, window, st)
                      : fork_commit_dispatch<__nv_bfloat16, 64>(
                            f, chosen, max_rows, budget, window, st);
  return c.d == 128
             ? fork_commit_dispatch<float, 128>(f, chosen, max_rows, budget,
                                                window, st)
             : fork_commit_dispatch<float, 64>(f, chosen, max_rows, budget,
                                               window, st);
}

}  // namespace kvr
