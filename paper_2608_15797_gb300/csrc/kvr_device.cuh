// kvr_device.cuh -- small device helpers shared by the generic and the
// candidate kernels of libkvr (not part of the ABI).
#pragma once

#include <cuda_bf16.h>
#include <stdint.h>

namespace kvr {
namespace dev {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kMaxG = 8;

__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(__nv_bfloat16 x) {
  return __bfloat162float(x);
}

__device__ __forceinline__ float2 ld2(const float *p) {
  return *reinterpret_cast<const float2 *>(p);
}
__device__ __forceinline__ float2 ld2(const __nv_bfloat16 *p) {
  return __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(p));
}

__device__ __forceinline__ void st1(float *p, float x) { *p = x; }
__device__ __forceinline__ void st1(__nv_bfloat16 *p, float x) {
  *p = __float2bfloat16_rn(x);
}

__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}
__device__ __forceinline__ float warp_max(float x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1)
    x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, o));
  return x;
}

// Collect, in index order, the indices i in [lo, hi) with pred(i) into list.
// Every thread of the block must call it; returns the count.
template <typename Pred>
__device__ int block_collect(int lo, int hi, Pred pred, int *list,
                             int *s_wsum, int *s_base) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (tid == 0) *s_base = 0;
  __syncthreads();
  for (int base = lo; base < hi; base += kThreads) {
    const int i = base + tid;
    const bool f = i < hi && pred(i);
    const unsigned bal = __ballot_sync(0xffffffffu, f);
    if (lane == 0) s_wsum[warp] = __popc(bal);
    __syncthreads();
    int off = *s_base;
    for (int w = 0; w < warp; ++w) off += s_wsum[w];
    if (f) list[off + __popc(bal & ((1u << lane) - 1u))] = i;
    __syncthreads();
    if (tid == 0) {
      int tot = 0;
      for (int w = 0; w < kWarps; ++w) tot += s_wsum[w];
      *s_base += tot;
    }
    __syncthreads();
  }
  const int total = *s_base;
  __syncthreads();  // every thread has read the count before it is reused
  return total;
}

// A float's order as an unsigned integer, negative values included.
__device__ __forceinline__ unsigned ord_bits(float z) {
  const unsigned b = __float_as_uint(z);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// R-KV key: higher z first, then lower position.
__device__ __forceinline__ unsigned long long rkv_key(float z, int32_t p) {
  return (static_cast<unsigned long long>(ord_bits(z)) << 32) |
         static_cast<unsigned long long>(0xFFFFFFFFu - static_cast<unsigned>(p));
}

// TopB key: higher score first, then lower position (scores are >= 0, so
// their IEEE bit patterns order like the values).
__device__ __forceinline__ unsigned long long rank_key(float s, int32_t p) {
  return ((unsigned long long)__float_as_uint(s) << 32) |
         (unsigned long long)(0xFFFFFFFFu - (unsigned)p);
}

// Block radix select (8 passes of 8 bits): the need-th largest rank_key among
// the rows i in [0, n) with cand(i).  Every thread must call it; all get the
// same key.  need >= 1 and at least `need` candidates must exist.
template <typename Cand, typename Key>
__device__ unsigned long long block_select(int n, int need, Cand cand, Key key,
                                           unsigned *hist,
                                           unsigned long long *s_prefix,
                                           int *s_need) {
  const int tid = threadIdx.x;
  unsigned long long prefix = 0, mask = 0;
  for (int shift = 56; shift >= 0; shift -= 8) {
    for (int i = tid; i < 256; i += kThreads) hist[i] = 0;
    __syncthreads();
    for (int i = tid; i < n; i += kThreads) {
      if (cand(i)) {
        const unsigned long long k = key(i);
        if ((k & mask) == prefix) atomicAdd(&hist[(k >> shift) & 255], 1u);
      }
    }
    __syncthreads();
    if (tid == 0) {
      int cnt = 0, dg = 255;
      for (; dg > 0; --dg) {
        if (cnt + (int)hist[dg] >= need) break;
        cnt += (int)hist[dg];
      }
      *s_prefix = prefix | ((unsigned long long)dg << shift);
      *s_need = need - cnt;
    }
    __syncthreads();
    prefix = *s_prefix;
    need = *s_need;
    mask |= 0xFFull << shift;
    __syncthreads();
  }
  return prefix;
}

// TopB by rank for units of at most kThreads rows, one row per thread: row
// i is kept iff it is not a candidate, or fewer than `need` candidates have
// a larger key (keys of candidates are distinct and nonzero).  Every thread
// must call it; s_keep[i] holds the answer for i < n afterwards.
template <typename Cand, typename Key>
__device__ void block_rank_keep(int n, int need, Cand cand, Key key,
                                unsigned long long *s_key,
                                unsigned char *s_keep) {
  const int i = threadIdx.x;
  const bool ci = i < n && cand(i);
  if (i < n) s_key[i] = ci ? key(i) : 0ull;
  __syncthreads();
  if (i < n) {
    bool k = true;
    if (ci) {
      const unsigned long long ki = s_key[i];
      int above = 0;
      for (int j = 0; j < n; ++j) above += s_key[j] > ki ? 1 : 0;
      k = above < need;
    }
    s_keep[i] = k ? 1 : 0;
  }
  __syncthreads();
}

}  // namespace dev
}  // namespace kvr
