// kvr_entropy.cu -- the entropy test of the online degeneration detector
// (Sec. 3.2, "Incoherent generation"; App. C, "Online degeneration
// detection") and its C ABI (include/kvr.h, kvr_entropy_*).
//
// One launch per generated token screens every candidate row:
//   H_e = -sum_v p_e(v) ln p_e(v), p_e = softmax(logits / T) over the whole
//   vocabulary, then the moving mean over the last min(e, window) tokens and
//   the stop test (e > guard and mean > tau).
//
// The work is one read of every logit, so the kernel is an HBM stream.
// `entropy_stream_kernel` (rows 16-byte aligned) is persistent: a multiple of
// the SM count of CTAs (three a SM), each streaming one contiguous, equal
// span of the [rows][vocab] logits.  In each CTA one producer thread moves
// 16 KB stages into a four-stage shared-memory ring with cp.async.bulk
// (completion on an mbarrier) and eight consumer warps reduce them, so HBM
// reads and the arithmetic overlap.  `entropy_kernel` (any alignment) cuts each row into
// pieces of 2,048 16-byte vectors (16,384 bf16 or 8,192 fp32 logits), one
// CTA each.  Both keep an online softmax in base 2:
//   y = x * log2(e) / T,  m = max y,  s = sum 2^(y - m),
//   t = sum 2^(y - m) (y - m),  so that  H = ln 2 * (log2 s - t / s).
// Every term of t has the same sign, so H is a sum of two non-negative
// terms with no cancellation.  A CTA merges its threads' (m, s, t) in a fixed
// shuffle tree at the end of each row segment it holds; the last CTA of a row
// to finish (an arrival counter per row, reset by that CTA) merges the row's
// segments in order, so the result does not depend on scheduling, and
// updates the row's state: the ring of entropies, the token count and the
// stop position.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <vector>

#include "../../include/kvr.h"
#include "kvr_internal.h"
#include "kvr_ptx.cuh"

namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kUnroll = 8;                        // 16-byte loads in flight
constexpr int kPieceVecs = kThreads * kUnroll;    // vectors per CTA
constexpr int kMaxWindow = 64;
constexpr float kLn2 = 0.693147180559945309f;
constexpr float kFloorExp = -128.f;  // 2^-128 flushes to zero in ex2.ftz

constexpr int kGridMax = 1024;  // CTAs of the persistent kernel, at most

struct EntropyView {
  float *hist;       // [rows][window] ring of entropies
  int32_t *count;    // [rows] tokens seen since the row's reset
  int32_t *stop;     // [rows] stop position, 0 while live
  unsigned *ticket;  // [rows] pieces of the current launch that finished
  float4 *part;      // [rows][seg_stride] (m, s, t, bad) of each segment
  unsigned *err;     // device error word
  int rows, vocab, window, guard, pieces, seg_stride;
  float tau, c;      // c = log2(e) / temperature
};

struct StepIO {
  const void *logits;
  long long stride;  // elements between rows
  float *entropy, *mean;
  int32_t *stopped;
};

// Packed fp32 pairs (sm_100 and later): one instruction adds or fuses two
// lanes' worth of arithmetic.
__device__ __forceinline__ uint64_t pk(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void upk(uint64_t v, float &lo, float &hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t fma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.ftz.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t add2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.ftz.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

__device__ __forceinline__ float max_nan(float a, float b) {
  float r;
  asm("max.NaN.f32 %0, %1, %2;" : "=f"(r) : "f"(a), "f"(b));
  return r;
}

// Per-thread online state over raw logits.  The sums are relative to the
// reference m = mx * c (rounded once, the same m for every term), where mx
// is one of the logits seen:
//  - add() keeps mx the largest logit seen, with a rescale when it grows,
//    and turns -inf logits into exact zero terms;
//  - add_fast() keeps the current reference (no maximum, no floor), so a
//    logit above mx gives a term above 1.  Terms stay finite while the
//    logits are finite and within about 88 / c of mx, and the sums keep full
//    relative precision at any scale.  The caller checks finite() after a
//    batch and redoes it with add() from the saved state if a term
//    overflowed or a logit was -inf, +inf or NaN.
struct Online {
  float mx = -INFINITY, s = 0.f, t = 0.f;
  bool bad = false;  // a NaN or +inf logit was seen

  template <int N>
  __device__ __forceinline__ void add(const float (&x)[N], float c) {
    float cm = x[0];
#pragma unroll
    for (int j = 1; j < N; ++j) cm = max_nan(cm, x[j]);
    bad |= (cm != cm) | (cm == INFINITY);
    if (cm > mx) {
      if (s > 0.f) {
        const float dd = mx * c - cm * c;  // <= 0
        const float f = kvr::ptx::ex2(dd);
        t = f * fmaf(dd, s, t);
        s *= f;
      }
      mx = cm;
    }
    const float nm = -(mx * c);
#pragma unroll
    for (int j = 0; j < N; ++j) {
      // -inf logits (masked tokens) give d = -inf or NaN; the floor turns
      // either into an exact zero term.
      const float d = fmaxf(fmaf(x[j], c, nm), kFloorExp);
      const float e = kvr::ptx::ex2(d);
      s += e;
      t = fmaf(e, d, t);
    }
  }

  // Terms in pairs with packed fp32 arithmetic: the pair sums (even and
  // odd terms) are added into s and t at the end.
  template <int N>
  __device__ __forceinline__ void add_fast(const float (&x)[N], float c,
                                           float nm) {
    static_assert(N % 2 == 0, "pairs");
    const uint64_t cc = pk(c, c), mm = pk(nm, nm);
    uint64_t s2 = pk(0.f, 0.f), t2 = pk(0.f, 0.f);
#pragma unroll
    for (int j = 0; j < N; j += 2) {
      const uint64_t d = fma2(pk(x[j], x[j + 1]), cc, mm);
      float d0, d1;
      upk(d, d0, d1);
      const uint64_t e = pk(kvr::ptx::ex2(d0), kvr::ptx::ex2(d1));
      s2 = add2(s2, e);
      t2 = fma2(e, d, t2);
    }
    float s0, s1, t0, t1;
    upk(s2, s0, s1);
    upk(t2, t0, t1);
    s += s0 + s1;
    t += t0 + t1;
  }

  __device__ __forceinline__ bool finite() const {
    return fabsf(s) < INFINITY && fabsf(t) < INFINITY;
  }
};

template <bool kBf16>
__device__ __forceinline__ void to_float(const uint4 &w,
                                         float (&x)[kBf16 ? 8 : 4]) {
  if constexpr (kBf16) {
    const uint32_t u[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      x[2 * j] = __uint_as_float(u[j] << 16);
      x[2 * j + 1] = __uint_as_float(u[j] & 0xffff0000u);
    }
  } else {
    x[0] = __uint_as_float(w.x), x[1] = __uint_as_float(w.y);
    x[2] = __uint_as_float(w.z), x[3] = __uint_as_float(w.w);
  }
}

// Add the vectors v[k] (k < K, those with ok[k]) to acc: the fast path,
// with the careful path redoing the batch on a non-finite result.  A thread
// with no reference yet takes the largest logit of its first vector.
template <bool kBf16, int K>
__device__ __forceinline__ void add_vectors(Online &acc, const uint4 (&v)[K],
                                            const bool (&ok)[K], float c) {
  constexpr int kPer = kBf16 ? 8 : 4;
  if (!(fabsf(acc.mx) < INFINITY) && ok[0]) {
    float x[kPer];
    to_float<kBf16>(v[0], x);
    float cm = x[0];
#pragma unroll
    for (int j = 1; j < kPer; ++j) cm = fmaxf(cm, x[j]);
    if (fabsf(cm) < INFINITY) acc.mx = cm;
  }
  if (fabsf(acc.mx) < INFINITY) {
    const float mx0 = acc.mx, s0 = acc.s, t0 = acc.t;
    const float nm = -(acc.mx * c);
#pragma unroll
    for (int k = 0; k < K; ++k) {
      if (ok[k]) {
        float x[kPer];
        to_float<kBf16>(v[k], x);
        acc.add_fast(x, c, nm);
      }
    }
    if (acc.finite()) return;
    acc.mx = mx0, acc.s = s0, acc.t = t0;
  }
#pragma unroll
  for (int k = 0; k < K; ++k) {
    if (ok[k]) {
      float x[kPer];
      to_float<kBf16>(v[k], x);
      acc.add(x, c);
    }
  }
}

// (m, s, t) with m the scaled reference; an empty partial has s = 0.
__device__ __forceinline__ void merge(float &m, float &s, float &t, float m2,
                                      float s2, float t2) {
  if (!(s2 > 0.f)) return;
  if (!(s > 0.f)) {
    m = m2, s = s2, t = t2;
    return;
  }
  const float M = fmaxf(m, m2);
  const float d1 = m - M, d2 = m2 - M;
  const float f1 = kvr::ptx::ex2(d1), f2 = kvr::ptx::ex2(d2);
  t = f1 * fmaf(d1, s, t) + f2 * fmaf(d2, s2, t2);
  s = f1 * s + f2 * s2;
  m = M;
}

// Merge the 32 lanes' (m, s, t): every lane moves its sums to the warp's
// largest reference M (one rescale), then plain sums.  Same result as
// pairwise merges up to rounding order, which is fixed.
__device__ __forceinline__ void warp_merge(float &m, float &s, float &t,
                                           unsigned &bad) {
  float M = s > 0.f ? m : -INFINITY;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1)
    M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
  if (s > 0.f) {
    const float d = m - M;  // <= 0
    const float f = kvr::ptx::ex2(d);
    t = f * fmaf(d, s, t);
    s *= f;
  } else {
    s = 0.f, t = 0.f;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    s += __shfl_xor_sync(0xffffffffu, s, o);
    t += __shfl_xor_sync(0xffffffffu, t, o);
  }
  bad = __reduce_or_sync(0xffffffffu, bad);
  m = M > -INFINITY ? M : 0.f;
}

template <bool kBf16>
__device__ __forceinline__ float load_one(const void *row, int i) {
  if (kBf16)
    return __bfloat162float(
        __ldcs(reinterpret_cast<const __nv_bfloat16 *>(row) + i));
  return __ldcs(reinterpret_cast<const float *>(row) + i);
}

// The row's state after its token: ring, count, stop; outputs.
__device__ void finish_row(const EntropyView &v, const StepIO &io, int r,
                           float m, float s, float t, bool bad) {
  (void)m;
  float H;
  if (bad || !(s > 0.f) || !isfinite(s) || !isfinite(t)) {
    H = __int_as_float(0x7fc00000);  // NaN
    atomicOr(v.err, kvr::ERR_NONFINITE);
  } else {
    H = kLn2 * (log2f(s) - t / s);
  }
  const int W = v.window;
  const int e = v.count[r] + 1;
  v.count[r] = e;
  float *h = v.hist + static_cast<size_t>(r) * W;
  h[(e - 1) % W] = H;
  const int n = min(e, W);
  float acc = 0.f;
  for (int i = 0; i < n; ++i) acc += h[(e - n + i) % W];
  const float mean = acc / static_cast<float>(n);
  int st = 0;
  if (e > v.guard && acc > v.tau * static_cast<float>(n)) {
    st = e;
    v.stop[r] = e;
  }
  if (io.entropy) io.entropy[r] = H;
  if (io.mean) io.mean[r] = mean;
  if (io.stopped) io.stopped[r] = st;
}

// grid (pieces, rows); kVec: 16-byte aligned rows read as vectors.
template <bool kBf16, bool kVec>
__global__ void __launch_bounds__(kThreads, 4)
    entropy_kernel(const EntropyView v, const StepIO io) {
  kvr::pdl_begin();
  __shared__ float4 s_warp[kWarps];
  const int p = blockIdx.x, r = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

  if (v.stop[r] != 0) {  // stopped before this token: nothing is read
    if (p == 0 && tid == 0) {
      if (io.entropy) io.entropy[r] = __int_as_float(0x7fc00000);
      if (io.mean) io.mean[r] = __int_as_float(0x7fc00000);
      if (io.stopped) io.stopped[r] = v.stop[r];
    }
    return;
  }

  constexpr int kPer = kBf16 ? 8 : 4;  // logits per 16-byte vector
  const char *row = static_cast<const char *>(io.logits) +
                    static_cast<long long>(r) * io.stride * (kBf16 ? 2 : 4);
  const float c = v.c;
  Online acc;
  const int piece_elems = kPieceVecs * kPer;
  const int e0 = p * piece_elems;
  const int e1 = min(v.vocab, e0 + piece_elems);
  if (kVec) {
    const uint4 *vec = reinterpret_cast<const uint4 *>(row);
    const int nvec = v.vocab / kPer;
    const int v0 = p * kPieceVecs;
    uint4 w[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int i = v0 + tid + u * kThreads;
      w[u] = i < nvec ? __ldcs(vec + i) : make_uint4(0, 0, 0, 0);
    }
    {
      bool ok[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) ok[u] = v0 + tid + u * kThreads < nvec;
      add_vectors<kBf16, kUnroll>(acc, w, ok, c);
    }
    // logits past the last whole vector belong to the last piece
    if (p == v.pieces - 1) {
      for (int i = nvec * kPer + tid; i < v.vocab; i += kThreads) {
        const float x[1] = {load_one<kBf16>(row, i)};
        acc.add(x, c);
      }
    }
  } else {
    for (int i = e0 + tid; i < e1; i += kThreads) {
      const float x[1] = {load_one<kBf16>(row, i)};
      acc.add(x, c);
    }
  }

  float m = acc.s > 0.f ? acc.mx * c : 0.f, s = acc.s, t = acc.t;
  unsigned bad = acc.bad ? 1u : 0u;
  warp_merge(m, s, t, bad);
  if (lane == 0) s_warp[warp] = make_float4(m, s, t, __uint_as_float(bad));
  __syncthreads();
  if (warp != 0) return;
  {
    const float4 q = lane < kWarps ? s_warp[lane] : make_float4(0, 0, 0, 0);
    m = q.x, s = q.y, t = q.z;
    bad = lane < kWarps ? __float_as_uint(q.w) : 0u;
    warp_merge(m, s, t, bad);
  }
  if (v.pieces == 1) {
    if (lane == 0) finish_row(v, io, r, m, s, t, bad != 0);
    return;
  }
  int last = 0;
  if (lane == 0) {
    v.part[static_cast<size_t>(r) * v.seg_stride + p] =
        make_float4(m, s, t, __uint_as_float(bad));
    __threadfence();
    last = atomicAdd(v.ticket + r, 1u) == static_cast<unsigned>(v.pieces - 1);
  }
  if (!__shfl_sync(0xffffffffu, last, 0)) return;
  __threadfence();
  // Last piece of the row: merge the pieces in piece order.
  m = 0.f, s = 0.f, t = 0.f, bad = 0u;
  const float4 *pr = v.part + static_cast<size_t>(r) * v.seg_stride;
  for (int i = lane; i < v.pieces; i += 32) {
    const float4 q = __ldcg(pr + i);
    merge(m, s, t, q.x, q.y, q.z);
    bad |= __float_as_uint(q.w);
  }
  warp_merge(m, s, t, bad);
  if (lane == 0) {
    v.ticket[r] = 0u;
    finish_row(v, io, r, m, s, t, bad != 0);
  }
}

// ---- persistent streaming kernel ------------------------------------------

constexpr int kSWarps = 8;                    // consumer warps
constexpr int kSThreads = (kSWarps + 1) * 32;  // + one producer warp
constexpr int kStageVecs = 1024;              // 16 KB a stage
constexpr int kSStages = 4;                   // three CTAs fit an SM
static_assert(kStageVecs % (kSWarps * 32) == 0,
              "every consumer thread takes the same number of vectors");
constexpr size_t kStreamSmem =
    static_cast<size_t>(kSStages) * kStageVecs * 16 + kSStages * 16 +
    2 * kSStages * 8;
enum : int { F_SEG_END = 1, F_ROW_END = 2, F_DONE = 4 };

__device__ __forceinline__ void named_sync_consumers() {
  asm volatile("bar.sync 1, %0;" ::"n"(kSWarps * 32) : "memory");
}

// Lane 0 of warp 0 holds the CTA's (m, s, t, bad) for its segment of row r:
// store it, or, as the row's last segment to arrive, merge them all.
__device__ void segment_done(const EntropyView &v, const StepIO &io, int r,
                             int nvf, long long span, float m, float s,
                             float t, unsigned bad, int lane) {
  const long long r0 = static_cast<long long>(r) * nvf;
  const int first = static_cast<int>(r0 / span);
  const int nseg = static_cast<int>((r0 + nvf - 1) / span) - first + 1;
  if (nseg == 1) {
    if (lane == 0) finish_row(v, io, r, m, s, t, bad != 0);
    return;
  }
  float4 *pr = v.part + static_cast<size_t>(r) * v.seg_stride;
  int last = 0;
  if (lane == 0) {
    pr[blockIdx.x - first] = make_float4(m, s, t, __uint_as_float(bad));
    __threadfence();
    last = atomicAdd(v.ticket + r, 1u) == static_cast<unsigned>(nseg - 1);
  }
  if (!__shfl_sync(0xffffffffu, last, 0)) return;
  __threadfence();
  m = 0.f, s = 0.f, t = 0.f, bad = 0u;
  for (int i = lane; i < nseg; i += 32) {
    const float4 q = __ldcg(pr + i);
    merge(m, s, t, q.x, q.y, q.z);
    bad |= __float_as_uint(q.w);
  }
  warp_merge(m, s, t, bad);
  if (lane == 0) {
    v.ticket[r] = 0u;
    finish_row(v, io, r, m, s, t, bad != 0);
  }
}

// grid: persistent CTAs; CTA b streams vectors [b * span, (b + 1) * span) of
// the rows' concatenated whole 16-byte vectors (nvf a row); a row's last
// vocab % (16 / element size) logits go with the segment holding its last
// whole vector.
template <bool kBf16>
__global__ void __launch_bounds__(kSThreads, 3)
    entropy_stream_kernel(const EntropyView v, const StepIO io,
                          const long long span, const int nvf) {
  using namespace kvr::ptx;
  kvr::pdl_begin();
  extern __shared__ __align__(128) unsigned char smem[];
  uint4 *data = reinterpret_cast<uint4 *>(smem);
  int4 *hdr = reinterpret_cast<int4 *>(smem + kSStages * kStageVecs * 16);
  uint64_t *full = reinterpret_cast<uint64_t *>(hdr + kSStages);
  uint64_t *empty = full + kSStages;
  __shared__ float4 s_warp[2][kSWarps];
  __shared__ int s_abort, s_issued, s_waited;
  constexpr int kPer = kBf16 ? 8 : 4;
  constexpr int kEs = kBf16 ? 2 : 4;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (tid == 0) {
    for (int q = 0; q < kSStages; ++q) {
      mbar_init(smem_u32(&full[q]), 1);
      mbar_init(smem_u32(&empty[q]), kSWarps);
    }
    s_abort = 0, s_issued = 0, s_waited = 0;
    fence_mbar_init();
  }
  __syncthreads();
  const long long total = static_cast<long long>(v.rows) * nvf;
  const long long b0 = static_cast<long long>(blockIdx.x) * span;
  const long long b1 = min(total, b0 + span);
  const char *base = static_cast<const char *>(io.logits);
  const size_t row_bytes = static_cast<size_t>(io.stride) * kEs;
  volatile int *abort = &s_abort;

  if (warp == kSWarps) {
    // Producer: one thread walks the span row by row in stages.
    if (lane == 0) {
      int q = 0;
      bool ok = true;
      for (long long f = b0; ok && f < b1;) {
        const int r = static_cast<int>(f / nvf);
        int a = static_cast<int>(f - static_cast<long long>(r) * nvf);
        const long long row_end = static_cast<long long>(r + 1) * nvf;
        const long long seg_end = min(b1, row_end);
        if (v.stop[r] != 0) {  // stopped earlier: not read
          if (a == 0) {
            if (io.entropy) io.entropy[r] = __int_as_float(0x7fc00000);
            if (io.mean) io.mean[r] = __int_as_float(0x7fc00000);
            if (io.stopped) io.stopped[r] = v.stop[r];
          }
          f = seg_end;
          continue;
        }
        int left = static_cast<int>(seg_end - f);
        while (left > 0) {
          const int n = min(left, kStageVecs);
          const int st = q % kSStages;
          const uint32_t ph = static_cast<uint32_t>(q / kSStages) & 1u;
          if (!mbar_wait(smem_u32(&empty[st]), ph ^ 1u, abort)) {
            atomicOr(v.err, kvr::ERR_TIMEOUT);
            *abort = 1;
            ok = false;
            break;
          }
          const int flags = left == n ? F_SEG_END | (seg_end == row_end
                                                         ? F_ROW_END : 0)
                                      : 0;
          hdr[st] = make_int4(r, a, n, flags);
          mbar_expect_tx(smem_u32(&full[st]), static_cast<uint32_t>(n) * 16u);
          bulk_load(smem_u32(data + st * kStageVecs),
                    base + r * row_bytes + static_cast<size_t>(a) * 16,
                    static_cast<uint32_t>(n) * 16u, smem_u32(&full[st]));
          ++q;
          *reinterpret_cast<volatile int *>(&s_issued) = q;
          a += n;
          left -= n;
        }
        f = seg_end;
      }
      if (ok) {  // terminator: a stage with no data
        const int st = q % kSStages;
        const uint32_t ph = static_cast<uint32_t>(q / kSStages) & 1u;
        if (mbar_wait(smem_u32(&empty[st]), ph ^ 1u, abort)) {
          hdr[st] = make_int4(0, 0, 0, F_DONE);
          mbar_arrive(smem_u32(&full[st]));
        } else {
          atomicOr(v.err, kvr::ERR_TIMEOUT);
          *abort = 1;
        }
      }
    }
  } else {
    // Consumers: eight warps reduce each stage from shared memory.
    const float c = v.c;
    Online acc;
    int segs = 0;
    for (int q = 0;; ++q) {
      const int st = q % kSStages;
      const uint32_t ph = static_cast<uint32_t>(q / kSStages) & 1u;
      int got = 1;
      if (lane == 0) got = mbar_wait(smem_u32(&full[st]), ph, abort);
      got = __shfl_sync(0xffffffffu, got, 0);
      if (!got) {
        if (lane == 0) {
          atomicOr(v.err, kvr::ERR_TIMEOUT);
          *abort = 1;
        }
        break;
      }
      if (tid == 0) *reinterpret_cast<volatile int *>(&s_waited) = q + 1;
      const int4 h = hdr[st];
      if (h.w & F_DONE) break;
      const uint4 *src = data + st * kStageVecs;
      constexpr int kV = kStageVecs / (kSWarps * 32);
      uint4 w[kV];
      bool ok[kV];
#pragma unroll
      for (int k = 0; k < kV; ++k) {
        const int i = tid + k * kSWarps * 32;
        ok[k] = i < h.z;
        w[k] = ok[k] ? src[i] : make_uint4(0, 0, 0, 0);
      }
      add_vectors<kBf16, kV>(acc, w, ok, c);
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&empty[st]));
      if (h.w & F_ROW_END) {
        const char *row = base + h.x * row_bytes;
        for (int i = nvf * kPer + tid; i < v.vocab; i += kSWarps * 32) {
          const float x[1] = {load_one<kBf16>(row, i)};
          acc.add(x, c);
        }
      }
      if (h.w & F_SEG_END) {
        float m = acc.s > 0.f ? acc.mx * c : 0.f, s = acc.s, t = acc.t;
        unsigned bad = acc.bad ? 1u : 0u;
        warp_merge(m, s, t, bad);
        if (lane == 0)
          s_warp[segs & 1][warp] = make_float4(m, s, t, __uint_as_float(bad));
        named_sync_consumers();
        if (warp == 0) {
          const float4 w4 = lane < kSWarps ? s_warp[segs & 1][lane]
                                           : make_float4(0.f, 0.f, 0.f, 0.f);
          m = w4.x, s = w4.y, t = w4.z;
          bad = lane < kSWarps ? __float_as_uint(w4.w) : 0u;
          warp_merge(m, s, t, bad);
          segment_done(v, io, h.x, nvf, span, m, s, t, bad, lane);
        }
        ++segs;
        acc = Online();
      }
    }
  }
  __syncthreads();
  // After an abort, wait (bounded) for copies still landing in the ring.
  if (s_abort && tid == 0) {
    volatile int never = 0;
    for (int q = s_waited; q < s_issued; ++q)
      mbar_wait(smem_u32(&full[q % kSStages]),
                static_cast<uint32_t>(q / kSStages) & 1u, &never);
  }
}

__global__ void entropy_reset_kernel(const EntropyView v, int b, int e) {
  kvr::pdl_begin();
  const int r = b + blockIdx.x * blockDim.x + threadIdx.x;
  if (r < e) {
    v.count[r] = 0;
    v.stop[r] = 0;
  }
}

constexpr size_t kAlign = 256;
size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

bool desc_ok(const kvr_entropy_desc *d) {
  if (!d) return false;
  if (d->rows < 1 || d->rows > 65535 || d->vocab < 1) return false;
  if (d->window < 1 || d->window > kMaxWindow || d->guard < 0) return false;
  if (d->logits_dtype != KVR_BF16 && d->logits_dtype != KVR_F32) return false;
  if (!std::isfinite(d->tau)) return false;
  if (!(d->temperature >= 0.f) || !std::isfinite(d->temperature)) return false;
  return true;
}

int pieces_for(const kvr_entropy_desc *d) {
  const long long per = kPieceVecs * (d->logits_dtype == KVR_BF16 ? 8 : 4);
  return static_cast<int>((d->vocab + per - 1) / per);
}

// Partials a row can have: pieces of entropy_kernel, or segments of the
// persistent kernel (a span is at least rows * nvf / kGridMax vectors, so a
// row meets at most ceil(kGridMax / rows) + 1 of them).
int seg_stride_for(const kvr_entropy_desc *d) {
  return std::max(pieces_for(d), (kGridMax + d->rows - 1) / d->rows + 2);
}

struct Layout {
  size_t hist, count, stop, ticket, part, err, total;
};

Layout layout(const kvr_entropy_desc *d) {
  Layout L;
  const size_t R = d->rows;
  size_t o = 0;
  L.hist = o, o = align_up(o + R * d->window * sizeof(float));
  L.count = o, o = align_up(o + R * sizeof(int32_t));
  L.stop = o, o = align_up(o + R * sizeof(int32_t));
  L.ticket = o, o = align_up(o + R * sizeof(unsigned));
  L.part = o, o = align_up(o + R * seg_stride_for(d) * sizeof(float4));
  L.err = o, o = align_up(o + sizeof(unsigned));
  L.total = o;
  return L;
}

cudaStream_t as_stream(void *s) { return reinterpret_cast<cudaStream_t>(s); }

// Persistent grid: resident CTAs per SM x SMs, at most kGridMax.
cudaError_t stream_setup(int *grid) {
  int dev = 0, sms = 0, per_sm = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess)
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  for (auto kern : {entropy_stream_kernel<true>, entropy_stream_kernel<false>}) {
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               static_cast<int>(kStreamSmem));
  }
  if (e == cudaSuccess)
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(
        &per_sm, entropy_stream_kernel<true>, kSThreads, kStreamSmem);
  if (e != cudaSuccess) return e;
  *grid = std::max(1, std::min(kGridMax, sms * std::max(per_sm, 1)));
  return cudaSuccess;
}

kvr_status fail(kvr_status st, const char *msg) {
  return static_cast<kvr_status>(kvr::report_error(st, msg));
}

kvr_status cuda_fail(const char *where, cudaError_t e) {
  return static_cast<kvr_status>(kvr::report_cuda_error(where, e));
}

}  // namespace

struct kvr_entropy {
  kvr_entropy_desc d;
  EntropyView v;
  void *buf;
  size_t bytes;
  uint64_t launches = 0;
  int stream_grid = 0;  // persistent CTAs (0: not yet sized)
  int kernel = 0;       // 0 auto, 1 streaming, 2 pieces
};

extern "C" {

size_t kvr_entropy_required_bytes(const kvr_entropy_desc *desc) {
  return desc_ok(desc) ? layout(desc).total : 0;
}

kvr_status kvr_entropy_create(const kvr_entropy_desc *desc, void *dev_buf,
                              size_t bytes, void *stream, kvr_entropy **out) {
  if (!out) return fail(KVR_EINVAL, "null output handle");
  *out = nullptr;
  if (!desc_ok(desc)) return fail(KVR_EINVAL, "invalid entropy descriptor");
  if (!dev_buf || reinterpret_cast<uintptr_t>(dev_buf) % kAlign)
    return fail(KVR_EINVAL, "device buffer null or not 256-byte aligned");
  const Layout L = layout(desc);
  if (bytes < L.total) return fail(KVR_ENOMEM, "device buffer too small");
  cudaError_t e = cudaMemsetAsync(dev_buf, 0, L.total, as_stream(stream));
  if (e != cudaSuccess) return cuda_fail("kvr_entropy_create: memset", e);
  auto *h = new kvr_entropy;
  h->d = *desc;
  h->buf = dev_buf;
  h->bytes = bytes;
  char *b = static_cast<char *>(dev_buf);
  EntropyView &v = h->v;
  v.hist = reinterpret_cast<float *>(b + L.hist);
  v.count = reinterpret_cast<int32_t *>(b + L.count);
  v.stop = reinterpret_cast<int32_t *>(b + L.stop);
  v.ticket = reinterpret_cast<unsigned *>(b + L.ticket);
  v.part = reinterpret_cast<float4 *>(b + L.part);
  v.err = reinterpret_cast<unsigned *>(b + L.err);
  v.rows = desc->rows;
  v.vocab = desc->vocab;
  v.window = desc->window;
  v.guard = desc->guard;
  v.pieces = pieces_for(desc);
  v.seg_stride = seg_stride_for(desc);
  v.tau = desc->tau;
  const double T = desc->temperature > 0.f ? desc->temperature : 1.0;
  v.c = static_cast<float>(1.4426950408889634074 / T);
  *out = h;
  return KVR_OK;
}

kvr_status kvr_entropy_reset(kvr_entropy *det, int row_begin, int row_end,
                             void *stream) {
  if (!det) return fail(KVR_EINVAL, "null detector");
  if (row_begin < 0 || row_end > det->d.rows || row_begin > row_end)
    return fail(KVR_EINVAL, "row range outside [0, rows]");
  if (row_begin == row_end) return KVR_OK;
  const int n = row_end - row_begin;
  cudaError_t e = kvr::launch_pdl(entropy_reset_kernel, dim3((n + 255) / 256),
                                  dim3(256), 0, as_stream(stream), det->v,
                                  row_begin, row_end);
  if (e != cudaSuccess) return cuda_fail("kvr_entropy_reset", e);
  ++det->launches;
  return KVR_OK;
}

kvr_status kvr_entropy_step(kvr_entropy *det, const void *logits,
                            int64_t row_stride, float *entropy, float *mean,
                            int32_t *stopped, void *stream) {
  if (!det) return fail(KVR_EINVAL, "null detector");
  if (!logits) return fail(KVR_EINVAL, "null logits");
  if (row_stride < det->d.vocab) return fail(KVR_EINVAL, "row_stride < vocab");
  const bool bf16 = det->d.logits_dtype == KVR_BF16;
  const int es = bf16 ? 2 : 4;
  if (reinterpret_cast<uintptr_t>(logits) % es)
    return fail(KVR_EINVAL, "logits not aligned to their element size");
  const bool vec = reinterpret_cast<uintptr_t>(logits) % 16 == 0 &&
                   (row_stride * es) % 16 == 0;
  StepIO io{logits, static_cast<long long>(row_stride), entropy, mean,
            stopped};
  const dim3 grid(det->v.pieces, det->d.rows);
  cudaStream_t st = as_stream(stream);
  cudaError_t e;
  const int nvf = det->d.vocab / (bf16 ? 8 : 4);
  // Measured at 512 rows x 152,064 logits, the streaming kernel is the
  // faster one for both element types.
  const bool stream_k = det->kernel != 2;
  if (vec && nvf >= 1 && stream_k) {
    if (!det->stream_grid) {
      e = stream_setup(&det->stream_grid);
      if (e != cudaSuccess) return cuda_fail("kvr_entropy_step: setup", e);
    }
    const long long total = static_cast<long long>(det->d.rows) * nvf;
    long long G = std::min<long long>(det->stream_grid, (total + 255) / 256);
    G = std::max<long long>(G, 1);
    const long long span = (total + G - 1) / G;
    G = (total + span - 1) / span;
    e = bf16 ? kvr::launch_pdl(entropy_stream_kernel<true>, dim3(G),
                               dim3(kSThreads), kStreamSmem, st, det->v, io,
                               span, nvf)
             : kvr::launch_pdl(entropy_stream_kernel<false>, dim3(G),
                               dim3(kSThreads), kStreamSmem, st, det->v, io,
                               span, nvf);
    if (e != cudaSuccess) return cuda_fail("kvr_entropy_step", e);
    ++det->launches;
    return KVR_OK;
  }
  if (bf16)
    e = vec ? kvr::launch_pdl(entropy_kernel<true, true>, grid, dim3(kThreads),
                              0, st, det->v, io)
            : kvr::launch_pdl(entropy_kernel<true, false>, grid,
                              dim3(kThreads), 0, st, det->v, io);
  else
    e = vec ? kvr::launch_pdl(entropy_kernel<false, true>, grid,
                              dim3(kThreads), 0, st, det->v, io)
            : kvr::launch_pdl(entropy_kernel<false, false>, grid,
                              dim3(kThreads), 0, st, det->v, io);
  if (e != cudaSuccess) return cuda_fail("kvr_entropy_step", e);
  ++det->launches;
  return KVR_OK;
}

kvr_status kvr_entropy_export(kvr_entropy *det, float *host_hist,
                              int32_t *host_count, int32_t *host_stopped,
                              void *stream) {
  if (!det) return fail(KVR_EINVAL, "null detector");
  cudaError_t e = cudaStreamSynchronize(as_stream(stream));
  if (e != cudaSuccess) return cuda_fail("kvr_entropy_export: sync", e);
  const int R = det->d.rows, W = det->d.window;
  std::vector<float> ring(static_cast<size_t>(R) * W);
  std::vector<int32_t> cnt(R), stp(R);
  e = cudaMemcpy(ring.data(), det->v.hist, ring.size() * sizeof(float),
                 cudaMemcpyDeviceToHost);
  if (e == cudaSuccess)
    e = cudaMemcpy(cnt.data(), det->v.count, R * sizeof(int32_t),
                   cudaMemcpyDeviceToHost);
  if (e == cudaSuccess)
    e = cudaMemcpy(stp.data(), det->v.stop, R * sizeof(int32_t),
                   cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail("kvr_entropy_export: copy", e);
  for (int r = 0; r < R; ++r) {
    if (host_hist) {
      const int c = cnt[r], n = std::min(c, W);
      float *h = host_hist + static_cast<size_t>(r) * W;
      for (int i = 0; i < W; ++i)
        h[i] = i < n ? ring[static_cast<size_t>(r) * W + (c - n + i) % W] : 0.f;
    }
    if (host_count) host_count[r] = cnt[r];
    if (host_stopped) host_stopped[r] = stp[r];
  }
  return KVR_OK;
}

kvr_status kvr_entropy_sync_status(kvr_entropy *det, void *stream) {
  if (!det) return fail(KVR_EINVAL, "null detector");
  cudaError_t e = cudaStreamSynchronize(as_stream(stream));
  if (e != cudaSuccess) return cuda_fail("kvr_entropy_sync_status: sync", e);
  unsigned word = 0;
  e = cudaMemcpy(&word, det->v.err, sizeof word, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail("kvr_entropy_sync_status: read", e);
  if (!word) return KVR_OK;
  e = cudaMemset(det->v.err, 0, sizeof word);
  if (e != cudaSuccess) return cuda_fail("kvr_entropy_sync_status: clear", e);
  return fail(KVR_EDEVICE, "non-finite logits in a row (entropy is NaN)");
}

kvr_status kvr_entropy_set_kernel(kvr_entropy *det, int kernel) {
  if (!det) return fail(KVR_EINVAL, "null detector");
  if (kernel < 0 || kernel > 2) return fail(KVR_EINVAL, "kernel must be 0..2");
  det->kernel = kernel;
  return KVR_OK;
}

kvr_status kvr_entropy_launch_count(const kvr_entropy *det, uint64_t *count) {
  if (!det || !count) return fail(KVR_EINVAL, "null detector or count");
  *count = det->launches;
  return KVR_OK;
}

void kvr_entropy_destroy(kvr_entropy *det) { delete det; }

}  // extern "C"
