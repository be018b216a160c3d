// kvr_copy.cu -- copying whole sequences between caches: App. C's
// "Best-of-(N+N)" forks candidates by physically copying the accepted
// sequence's live (post-eviction) KV slots, and the chosen candidate becomes
// the persistent sequence.  With kvr_cache_copy_sequences a caller forks N
// candidates into a cache of candidate sequences, decodes them with eviction
// every token (the paper's own candidate mode), and copies the chosen one
// back.
//
// One CTA per (pair, layer, KV head) copies the unit's live rows [0, len) of
// K and V (rows are kept compacted in those slots), their scores and
// positions, and the unit's state.  The work is data movement, so HBM
// bounds it: 16-byte loads and stores, several in flight per thread.
#include <cuda_runtime.h>

#include "kvr_internal.h"

namespace kvr {
namespace {

constexpr int kThreads = 256;
constexpr int kUnroll = 4;

__device__ __forceinline__ void copy16(int4 *dst, const int4 *src, size_t n) {
  const size_t step = static_cast<size_t>(kThreads) * kUnroll;
  size_t i = threadIdx.x;
  for (; i + (kUnroll - 1) * kThreads < n; i += step) {
    int4 v[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) v[u] = __ldcs(src + i + u * kThreads);
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) dst[i + u * kThreads] = v[u];
  }
  for (; i < n; i += kThreads) dst[i] = __ldcs(src + i);
}

// grid (L * H, pairs)
__global__ void __launch_bounds__(kThreads)
    copy_seq_kernel(const CacheView dst, const CacheView src, const SeqPairs p,
                    int row_bytes) {
  pdl_begin();
  const int lh = blockIdx.x;
  const int i = blockIdx.y;
  const size_t us = static_cast<size_t>(p.src[i]) * src.L * src.H + lh;
  const size_t ud = static_cast<size_t>(p.dst[i]) * dst.L * dst.H + lh;
  const int n = src.state[4 * us];
  if (n < 0 || n > dst.cap) {  // the host checked this against its mirror
    if (threadIdx.x == 0) atomicOr(dst.err, ERR_LENGTH);
    return;
  }
  const size_t kb = static_cast<size_t>(row_bytes);
  const char *sk = static_cast<const char *>(src.K) + us * src.cap * kb;
  const char *sv = static_cast<const char *>(src.V) + us * src.cap * kb;
  char *dk = static_cast<char *>(dst.K) + ud * dst.cap * kb;
  char *dv = static_cast<char *>(dst.V) + ud * dst.cap * kb;
  const size_t n16 = static_cast<size_t>(n) * kb / 16;
  copy16(reinterpret_cast<int4 *>(dk), reinterpret_cast<const int4 *>(sk), n16);
  copy16(reinterpret_cast<int4 *>(dv), reinterpret_cast<const int4 *>(sv), n16);
  for (int r = threadIdx.x; r < n; r += kThreads) {
    dst.score[ud * dst.sstride + r] = src.score[us * src.sstride + r];
    dst.pos[ud * dst.sstride + r] = src.pos[us * src.sstride + r];
  }
  // Length and next position; the R-KV key sum is not copied, so the
  // copy's is marked stale.
  if (threadIdx.x < 4)
    dst.state[4 * ud + threadIdx.x] =
        threadIdx.x == 2 ? 0 : src.state[4 * us + threadIdx.x];
}

}  // namespace

cudaError_t launch_copy_seqs(const CacheView &dst, const CacheView &src,
                             const SeqPairs &p, int n_pairs, int row_bytes,
                             cudaStream_t st) {
  if (n_pairs <= 0) return cudaSuccess;
  return launch_pdl(copy_seq_kernel, dim3(src.L * src.H, n_pairs),
                    dim3(kThreads), 0, st, dst, src, p, row_bytes);
}

}  // namespace kvr
