// kvr_fused.cu -- the fused steady-state decode step for bf16, head_dim 128,
// G <= 8 and at most 160 live rows per unit: append + Attn(q_t, C) (Eq. 1)
// + accumulated-attention update (Sec. 2.1) + TopB eviction of the single
// surplus row (Eq. 1 with the Sec. 4.1 window) + in-place compaction, in one
// pass over K and V.
//
// Design (GB300, sm_103a):
//  - Persistent CTAs, one per SM.  Each CTA owns a ring of shared-memory
//    stages; two producer warps fill a stage with one unit's K and V (two
//    128B-swizzled TMA boxes each: columns 0-63 and 64-127, all rows of the
//    unit), completing on the stage's mbarrier.  Consumer groups of U warps
//    each take whole units; within a group every warp owns one or two
//    16-row tiles of the unit (kvr_fused_unit.cuh).
//  - The small per-unit inputs (the G query rows, the new k/v row, scores,
//    positions and state) are fetched by the producer warp's 32 lanes with
//    16-byte cp.async copies that arrive on the same mbarrier, so a stage
//    costs the TMA unit only its four K/V boxes and the query rows land at
//    a padded pitch that keeps the ldmatrix reads free of bank conflicts.
//  - QK^T and PV run on warp-level bf16 tensor-core MMAs (m16n8k16, fp32
//    accumulate): K rows are the M side, the <= 8 query heads of the group
//    the N side.  The probability tile leaves the QK accumulators in
//    registers and becomes the PV B operand through movmatrix (an 8x8
//    transpose), so P never touches memory.  Softmax and score reductions
//    are warp shuffles.
//  - The new row is inserted into the staged tile, so K and V are read once
//    from HBM and nothing is re-read for the scores.  Exactly one row is
//    evicted (warp argmin of the (score, -position) key over non-window
//    rows) and the new row is written straight into the freed slot: the
//    compaction moves no other row.
//  - Units go to the groups round-robin, so when the ring depth is not a
//    multiple of the group count, one stage's consecutive units belong to
//    different groups and a group can reach a stage's next unit before the
//    previous one has landed.  A parity wait cannot tell those two phases
//    apart, so a group first waits until the producer has recorded the unit
//    as issued (which implies the earlier phase completed) and only then on
//    the stage's full barrier.
//  - Launched with programmatic stream serialization: a launch may start
//    while the previous kernel of the stream drains (its barrier setup
//    overlaps that tail); griddepcontrol.wait then holds every thread until
//    the previous grid has completed and its writes are visible, before the
//    first access to global memory.  Each CTA allows the next launch to
//    start once its own setup is done.
//  - Every wait on an mbarrier is bounded (about 2 s); on timeout the kernel
//    sets ERR_TIMEOUT in the device error word and drains its own copies.
#include <cuda.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "kvr_device.cuh"
#include "kvr_internal.h"
#include "kvr_ptx.cuh"

namespace kvr {
namespace {

using namespace ptx;

constexpr int kMaxStages = 8;
constexpr int kMaxTiles = 10;   // 16-row tiles a unit: at most 160 rows
constexpr int kMaxGroups = 4;      // units in flight on the consumer side
constexpr int kProducers = 2;      // TMA-issuing warps
constexpr int kMaxThreads = 512;   // consumer warps + the producers
constexpr int kQPitch = 272;  // bytes per staged query row (256 + 16 padding)

__device__ __forceinline__ void group_bar(int id, int threads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

// Byte offsets inside one stage of R staged rows (R a multiple of 16, so
// every box starts on a 1024-byte boundary as the 128B swizzle needs).
// The R-KV step also stages the unit's kept sum of normalised keys (rs,
// 128 fp32).
struct StageLayout {
  uint32_t k0, k1, v0, v1, q, kn, vn, sc, ps, st, rs, bytes;
  __host__ __device__ explicit StageLayout(int R, bool rkv = false) {
    k0 = 0;
    k1 = k0 + R * 128;
    v0 = k1 + R * 128;
    v1 = v0 + R * 128;
    q = v1 + R * 128;
    kn = q + 8 * kQPitch;
    vn = kn + 256;
    sc = vn + 256;
    ps = sc + 4 * R;
    st = ps + 4 * R;
    rs = st + 16;
    bytes = ((rs + (rkv ? 512 : 0)) + 1023) / 1024 * 1024;
  }
};

// Byte offsets inside one consumer group's private exchange area (after the
// ring): kSlots 16-byte slots per warp (five; six for the R-KV step), then
// the warps' partial outputs ([warp][8 head-dim tiles][32 lanes] float4).
// A one-warp group needs none.
struct GroupLayout {
  uint32_t xs, ox, bytes, slots;
  __host__ __device__ explicit GroupLayout(int U, bool rkv = false) {
    slots = rkv ? 6 : 5;
    xs = 0;
    ox = (U * slots * 16 + 127) / 128 * 128;
    // (the R-KV step also passes its parts of the key sum through the
    // partial-output area, one-warp groups included)
    bytes = (U > 1 || rkv) ? ox + U * 8 * 32 * 16 : 0;
  }
};

// Cache unit and input row of the launch's unit idx (sequence-major, then
// layer, then KV head).
struct UnitIdx {
  size_t ug;    // cache unit
  size_t krow;  // row of this unit in the call's [S][nl][H] inputs
};

__device__ __forceinline__ UnitIdx unit_idx(const FusedParams &p, int idx) {
  const int h = idx % p.c.H;
  const int lr = (idx / p.c.H) % p.nl;
  const int sq = idx / (p.c.H * p.nl);
  UnitIdx x;
  x.ug = ((size_t)sq * p.c.L + p.lb + lr) * p.c.H + h;
  x.krow = ((size_t)sq * p.nl + lr) * p.c.H + h;
  return x;
}

// Producer warp: enqueue one unit into a stage.  Lane 0 issues K and V as
// two 128B-swizzled TMA boxes of Rb rows each (columns 0-63, 64-127); all
// 32 lanes copy the small inputs in 16-byte pieces and arrive when theirs
// have landed (the full barrier expects 1 + 32 arrivals).
__device__ __forceinline__ void issue_unit(const FusedParams &p,
                                           const CUtensorMap *tmK,
                                           const CUtensorMap *tmV,
                                           unsigned char *stage, uint32_t bar,
                                           int idx, int lane) {
  const StageLayout L(p.R, p.rkv != 0);
  const UnitIdx x = unit_idx(p, idx);
  const uint32_t s0 = smem_u32(stage);
  if (lane == 0) {
    mbar_expect_tx(bar, 4u * p.Rb * 128u);
    const int row0 = (int)(x.ug * (size_t)p.c.cap);
    tma_load_2d(s0 + L.k0, tmK, 0, row0, bar);
    tma_load_2d(s0 + L.k1, tmK, 64, row0, bar);
    tma_load_2d(s0 + L.v0, tmV, 0, row0, bar);
    tma_load_2d(s0 + L.v1, tmV, 64, row0, bar);
  }
  const int G = p.c.G;
  const unsigned char *q =
      reinterpret_cast<const unsigned char *>(p.q + x.krow * G * 128);
  for (int i = lane; i < G * 16; i += 32)  // query rows, 16 pieces each
    cp_async16(s0 + L.q + (i >> 4) * kQPitch + (i & 15) * 16, q + i * 16);
  cp_async16(s0 + (lane < 16 ? L.kn : L.vn) + (lane & 15) * 16,
             reinterpret_cast<const unsigned char *>(
                 (lane < 16 ? p.k_new : p.v_new) + x.krow * 128) +
                 (lane & 15) * 16);
  const int nsc = p.Rb / 4;  // 16-byte pieces of the scores (and positions)
  const unsigned char *sc =
      reinterpret_cast<const unsigned char *>(p.c.score + x.ug * p.c.sstride);
  const unsigned char *ps =
      reinterpret_cast<const unsigned char *>(p.c.pos + x.ug * p.c.sstride);
  for (int i = lane; i < 2 * nsc; i += 32)
    cp_async16(s0 + (i < nsc ? L.sc + i * 16 : L.ps + (i - nsc) * 16),
               (i < nsc ? sc + i * 16 : ps + (i - nsc) * 16));
  if (lane == 31)
    cp_async16(s0 + L.st, p.c.state + x.ug * 4);
  if (p.rkv)  // the kept key sum (used only if the state marks it valid)
    cp_async16(s0 + L.rs + lane * 16,
               reinterpret_cast<const unsigned char *>(p.c.rsum + x.ug * 128) +
                   lane * 16);
  cp_async_arrive_noinc(bar);
}

#include "kvr_fused_unit.cuh"

static_assert(kDefaultWaitNs == kWaitNs, "one default wait bound");

// Bounded wait until the producer has recorded unit k (or a later one) as
// issued into this stage; false on timeout or abort.
__device__ bool wait_issued(volatile int *issued, int k, volatile int *abort,
                            uint64_t limit_ns) {
  if (*issued >= k) return true;
  const uint64_t t0 = global_ns();
  while (*issued < k) {
    if (*abort || global_ns() - t0 > limit_ns) return false;
  }
  return true;
}

template <int T, int U, bool kOutBf16, bool kRkv>
__global__ void __launch_bounds__(kMaxThreads, 1)
    fused_step_kernel(const __grid_constant__ CUtensorMap tmK,
                      const __grid_constant__ CUtensorMap tmV,
                      const FusedParams p) {
  extern __shared__ unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kMaxStages];
  __shared__ __align__(8) uint64_t empty_bar[kMaxStages];
  __shared__ volatile int issued_k[kMaxStages];
  __shared__ int consumed_k[kMaxStages];
  __shared__ volatile int s_abort;
  __shared__ volatile int s_ok[kMaxGroups];
  unsigned char *smem = reinterpret_cast<unsigned char *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_units = p.c.S * p.nl * p.c.H;
  const int mine = (int)blockIdx.x < n_units
                       ? (n_units - 1 - (int)blockIdx.x) / (int)gridDim.x + 1
                       : 0;
  const StageLayout L(16 * T, kRkv);
  const int consumers = p.n_groups * U;

  if (threadIdx.x == 0) {
    prefetch_tmap(&tmK);
    prefetch_tmap(&tmV);
    for (int s = 0; s < p.n_stages; ++s) {
      mbar_init(smem_u32(&full_bar[s]), 1 + 32);  // TMA + producer lanes
      mbar_init(smem_u32(&empty_bar[s]), U);  // one arrival per group warp
      issued_k[s] = -1;
      consumed_k[s] = -1;
    }
    s_abort = 0;
    fence_mbar_init();
  }
  // Query rows of heads >= G are never copied: zero them once per stage.
  for (int s = 0; s < p.n_stages; ++s) {
    unsigned char *q = smem + s * L.bytes + L.q;
    for (int i = threadIdx.x; i < (8 - p.c.G) * (kQPitch / 16);
         i += blockDim.x)
      reinterpret_cast<int4 *>(q + p.c.G * kQPitch)[i] = make_int4(0, 0, 0, 0);
  }
  fence_proxy_async();
  __syncthreads();
  pdl_begin();

  if (warp >= consumers) {
    // Producers: warp `consumers + j` owns the stages s with s % kProducers
    // == j, so every stage is refilled by one thread, round after round (two
    // threads on one stage could run a full ring ahead and alias the
    // mbarrier parity).
    const int j = warp - consumers;
    for (int k = 0; k < mine; ++k) {
      const int s = k % p.n_stages;
      if (s % kProducers != j) continue;
      // Test hook: the first unit of CTA 0 is never loaded (no copy is
      // issued, so there is nothing to drain); its group's wait runs out.
      if (p.c.hold_first && blockIdx.x == 0 && k == 0) continue;
      const uint32_t ph = (uint32_t)(k / p.n_stages) & 1u;
      // Lane 0 waits (bounded) and tells the warp; __syncwarp orders the
      // other lanes' copies after the consumers' release it observed.
      int ok = 1;
      if (lane == 0)
        ok = mbar_wait(smem_u32(&empty_bar[s]), ph ^ 1u, &s_abort, p.c.wait_ns);
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) {
        if (lane == 0) {
          atomicOr(p.c.err, ERR_TIMEOUT);
          s_abort = 1;
        }
        break;
      }
      __syncwarp();
      issue_unit(p, &tmK, &tmV, smem + s * L.bytes, smem_u32(&full_bar[s]),
                 (int)blockIdx.x + k * (int)gridDim.x, lane);
      __syncwarp();
      if (lane == 0) issued_k[s] = k;
    }
  } else if (warp < consumers) {
    const int grp = warp / U, w = warp % U, bar_id = 1 + grp;
    unsigned char *garea =
        smem + p.n_stages * L.bytes + grp * GroupLayout(U, kRkv).bytes;
    for (int k = grp; k < mine; k += p.n_groups) {
      const int s = k % p.n_stages;
      const uint32_t ph = (uint32_t)(k / p.n_stages) & 1u;
      // One warp waits (bounded) and tells the group, so that every warp
      // of the group takes the same branch before the next named barrier.
      if (w == 0) {
        const bool ok =
            wait_issued(&issued_k[s], k, &s_abort, p.c.wait_ns) &&
            mbar_wait(smem_u32(&full_bar[s]), ph, &s_abort, p.c.wait_ns);
        if (lane == 0) {
          s_ok[grp] = ok ? 1 : 0;
          if (!ok) {
            atomicOr(p.c.err, ERR_TIMEOUT);
            s_abort = 1;
          }
        }
      }
      group_bar(bar_id, 32 * U);
      if (!s_ok[grp]) break;
      mbar_try_wait(smem_u32(&full_bar[s]), ph);  // acquire for this thread
      UnitFront<(T + U - 1) / U> f;
      const bool ok = unit_front<T, U, kRkv>(
          p, smem + s * L.bytes, (int)blockIdx.x + k * (int)gridDim.x, w,
          lane, f, garea, bar_id);
      // Each warp releases the stage once its own reads and writes of it
      // are done (the async-proxy fence orders them before the refill); the
      // rest of the unit runs from registers and the group's own area.
      fence_proxy_async();
      __syncwarp();
      if (lane == 0) {
        if (w == 0) consumed_k[s] = k;
        mbar_arrive(smem_u32(&empty_bar[s]));
      }
      if (ok) {
        unit_publish<T, U, kRkv>(garea, f, w, lane);
        unit_back<T, U, kOutBf16, kRkv>(p, garea, f, w, lane, bar_id);
      }
    }
  }
  __syncthreads();
  // After an abort, wait (bounded) for copies still landing in our stages.
  if (s_abort && threadIdx.x == 0) {
    volatile int never = 0;
    for (int s = 0; s < p.n_stages; ++s) {
      const int k = issued_k[s];
      if (k >= 0 && consumed_k[s] != k)
        mbar_wait(smem_u32(&full_bar[s]), (uint32_t)(k / p.n_stages) & 1u,
                  &never);
    }
  }
}

template <int T, int U, bool kOutBf16, bool kRkv>
cudaError_t launch_tu(const CUtensorMap &tmK, const CUtensorMap &tmV,
                      const FusedParams &p, int grid, int smem_bytes,
                      cudaStream_t st) {
  auto kern = fused_step_kernel<T, U, kOutBf16, kRkv>;
  cudaError_t e = cudaFuncSetAttribute(
      kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes);
  if (e != cudaSuccess) return e;
  return launch_pdl(kern, dim3(grid), dim3(32 * (p.n_groups * U + kProducers)),
                    smem_bytes, st, tmK, tmV, p);
}

template <bool kOutBf16, bool kRkv>
cudaError_t launch_t(const CUtensorMap &tmK, const CUtensorMap &tmV,
                     const FusedParams &p, int grid, int smem_bytes,
                     cudaStream_t st) {
  // (tiles, warps per unit): one tile per warp, or two.
#define KVR_TU(T_, U_)                                                   \
  if (p.R == 16 * T_ && p.group_warps == U_)                             \
    return launch_tu<T_, U_, kOutBf16, kRkv>(tmK, tmV, p, grid,          \
                                             smem_bytes, st);
  KVR_TU(1, 1)
  KVR_TU(2, 1) KVR_TU(2, 2)
  KVR_TU(3, 2) KVR_TU(3, 3)
  KVR_TU(4, 2) KVR_TU(4, 4)
  KVR_TU(5, 3) KVR_TU(5, 5)
  KVR_TU(6, 3) KVR_TU(6, 6)
  KVR_TU(7, 4) KVR_TU(7, 7)
  KVR_TU(8, 4) KVR_TU(8, 8)
  KVR_TU(9, 5) KVR_TU(10, 5)
#undef KVR_TU
  return cudaErrorInvalidValue;
}

}  // namespace

int fused_stage_bytes(int R, bool rkv) {
  return (int)StageLayout(R, rkv).bytes;
}

int fused_group_warps(int R, int requested) {
  if (R % 16 != 0 || R < 16 || R > 16 * kMaxTiles) return 0;
  const int T = R / 16, one = T, two = (T + 1) / 2;
  // Past 8 tiles only two tiles a warp (one a warp would need 9-10 warps
  // a group; the register file holds two such groups at most).
  if (T > 8) return two;
  if (requested == one || requested == two) return requested;
  return T <= 3 ? one : two;  // measured: two tiles per warp from T = 4 on
}

int fused_group_bytes(int U, bool rkv) {
  return (int)GroupLayout(U, rkv).bytes;
}
int fused_max_groups() { return kMaxGroups; }
int fused_max_rows() { return 16 * kMaxTiles; }
int fused_max_threads() { return kMaxThreads; }
int fused_producer_warps() { return kProducers; }

cudaError_t launch_fused_step(const CUtensorMap &tmK, const CUtensorMap &tmV,
                              const FusedParams &p, int grid, int smem_bytes,
                              cudaStream_t st) {
  if (fused_group_warps(p.R, p.group_warps) != p.group_warps ||
      p.n_groups < 1 || p.n_groups > kMaxGroups || p.n_stages > kMaxStages ||
      32 * (p.n_groups * p.group_warps + kProducers) > kMaxThreads)
    return cudaErrorInvalidValue;
  if (p.rkv)
    return p.c.out_bf16
               ? launch_t<true, true>(tmK, tmV, p, grid, smem_bytes, st)
               : launch_t<false, true>(tmK, tmV, p, grid, smem_bytes, st);
  return p.c.out_bf16 ? launch_t<true, false>(tmK, tmV, p, grid, smem_bytes, st)
                      : launch_t<false, false>(tmK, tmV, p, grid, smem_bytes, st);
}

}  // namespace kvr
