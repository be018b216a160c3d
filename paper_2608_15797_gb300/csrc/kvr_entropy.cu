// kvr_entropy.cu -- the entropy test of the online degeneration detector
// (Sec. 3.3, "Incoherent generation"; App. Impl., "Online degeneration
// detection") and its C ABI (include/kvr.h, kvr_entropy_*).
//
// One launch per generated token screens every candidate row:
//   H_e = -sum_v p_e(v) ln p_e(v), p_e = softmax(logits / T) over the whole
//   vocabulary, then the moving mean over the last min(e, window) tokens and
//   the stop test (e > guard and mean > tau).
//
// The work is one read of every logit, so the kernel is an HBM stream.  Each
// row is cut into pieces of 2,048 16-byte vectors (16,384 bf16 or 8,192 fp32
// logits); one 256-thread CTA reads a piece with eight vector loads in
// flight per thread and keeps an online softmax in base 2:
//   y = x * log2(e) / T,  m = max y,  s = sum 2^(y - m),
//   t = sum 2^(y - m) (y - m),  so that  H = ln 2 * (log2 s - t / s).
// Every term of t has the same sign, so H is a sum of two non-negative
// terms with no cancellation.  A CTA merges its threads' (m, s, t) in a fixed
// shuffle tree; the last CTA of a row to finish (an arrival counter per row,
// reset by that CTA) merges the row's pieces in piece order, so the result
// does not depend on scheduling, and updates the row's state: the ring of
// entropies, the token count and the stop position.
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

struct EntropyView {
  float *hist;       // [rows][window] ring of entropies
  int32_t *count;    // [rows] tokens seen since the row's reset
  int32_t *stop;     // [rows] stop position, 0 while live
  unsigned *ticket;  // [rows] pieces of the current launch that finished
  float4 *part;      // [rows][pieces] (m, s, t, bad) of each piece
  unsigned *err;     // device error word
  int rows, vocab, window, guard, pieces;
  float tau, c;      // c = log2(e) / temperature
};

struct StepIO {
  const void *logits;
  long long stride;  // elements between rows
  float *entropy, *mean;
  int32_t *stopped;
};

__device__ __forceinline__ float max_nan(float a, float b) {
  float r;
  asm("max.NaN.f32 %0, %1, %2;" : "=f"(r) : "f"(a), "f"(b));
  return r;
}

// Per-thread online state over raw logits: mx is the largest logit seen, the
// sums are relative to m = mx * c (rounded once, the same m for every term).
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
};

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

__device__ __forceinline__ void warp_merge(float &m, float &s, float &t,
                                           unsigned &bad) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
    const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
    const float t2 = __shfl_xor_sync(0xffffffffu, t, o);
    bad |= __shfl_xor_sync(0xffffffffu, bad, o);
    merge(m, s, t, m2, s2, t2);
  }
}

__device__ __forceinline__ void unpack_bf16(const uint4 &w, float (&x)[8]) {
  const uint32_t u[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    x[2 * j] = __uint_as_float(u[j] << 16);
    x[2 * j + 1] = __uint_as_float(u[j] & 0xffff0000u);
  }
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
__global__ void __launch_bounds__(kThreads)
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
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      if (v0 + tid + u * kThreads < nvec) {
        float x[kPer];
        if constexpr (kBf16) {
          unpack_bf16(w[u], x);
        } else {
          x[0] = __uint_as_float(w[u].x), x[1] = __uint_as_float(w[u].y);
          x[2] = __uint_as_float(w[u].z), x[3] = __uint_as_float(w[u].w);
        }
        acc.add(x, c);
      }
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
    v.part[static_cast<size_t>(r) * v.pieces + p] =
        make_float4(m, s, t, __uint_as_float(bad));
    __threadfence();
    last = atomicAdd(v.ticket + r, 1u) == static_cast<unsigned>(v.pieces - 1);
  }
  if (!__shfl_sync(0xffffffffu, last, 0)) return;
  __threadfence();
  // Last piece of the row: merge the pieces in piece order.
  m = 0.f, s = 0.f, t = 0.f, bad = 0u;
  const float4 *pr = v.part + static_cast<size_t>(r) * v.pieces;
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
  L.part = o, o = align_up(o + R * pieces_for(d) * sizeof(float4));
  L.err = o, o = align_up(o + sizeof(unsigned));
  L.total = o;
  return L;
}

cudaStream_t as_stream(void *s) { return reinterpret_cast<cudaStream_t>(s); }

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

kvr_status kvr_entropy_launch_count(const kvr_entropy *det, uint64_t *count) {
  if (!det || !count) return fail(KVR_EINVAL, "null detector or count");
  *count = det->launches;
  return KVR_OK;
}

void kvr_entropy_destroy(kvr_entropy *det) { delete det; }

}  // extern "C"
