// kvr_chunked.cu -- the persistent decode step for units streamed in 32-row
// chunks: units longer than the staged kernel of kvr_fused.cu takes (the
// B = 128..512 sweep), and the candidate-batched step of stepwise best-of-N
// (Sec. 2.2 Eq. 2), where a job is one candidate of one unit and its rows are
// the parent's live rows (a shared, read-only prefix) followed by the
// candidate's private tail.  Append + Attn(q_t, C) (Eq. 1) + accumulated-
// attention update (Sec. 2.1, mean over the G heads) + for plain units the
// eviction of the single surplus row (TopB of Eq. 1 with the Sec. 4.1 window)
// and in-place compaction; for candidates the append to the private tail
// (eviction is deferred to the commit).  bf16, head_dim 128, G <= 8.
//
// Design (GB300, sm_103a):
//  - Persistent CTAs, one per SM.  A CTA runs n_groups independent consumer
//    groups of two warps, each with its own ring of n_stages chunk stages and
//    its own producer warp, so no group ever waits for another group's rows.
//  - A job's rows are segment A (plain units: none; candidates: the prefix,
//    from the parent slab) then segment B (the unit's rows, or the
//    candidate's tail) then the new row.  Each segment streams in chunks of
//    32 rows, loaded by TMA as 16-row 128B-swizzled boxes (so at most 15
//    rows past a segment's end are read); the new row is inserted into the
//    last chunk of B from the inputs.  The producer warp's 32 lanes fetch the
//    small inputs (query rows, new k/v row, old scores and positions of the
//    chunk) with cp.async onto the stage's mbarrier, and lane 0 writes a
//    chunk header (job, rows, flags) that the barrier releases.
//  - Each consumer warp owns one 16-row tile of every chunk: QK^T and PV on
//    bf16 mma.sync (m16n8k16, fp32 accumulate, P split hi + lo) with an
//    online softmax across the job's chunks, and it keeps the scaled logits,
//    old scores and positions of its rows in the group's area, then releases
//    the stage.  After the last chunk the two warps merge their softmax
//    states and partial outputs, compute every row's exact probability from
//    the kept logits for the score update, agree on the evicted row, and
//    write back.
//  - Launched with programmatic stream serialization; every mbarrier wait is
//    bounded (about 2 s) and on timeout sets ERR_TIMEOUT and drains its own
//    copies.
#include <cuda.h>
#include <cuda_bf16.h>
#include <math.h>
#include <stdint.h>

#include "kvr_internal.h"
#include "kvr_ptx.cuh"

namespace kvr {
namespace {

using namespace ptx;

// Packed fp32 pairs (round to nearest, no flush).
__device__ __forceinline__ uint64_t pk2(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void upk2(uint64_t v, float &lo, float &hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t mul2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

constexpr int kCR = 32;       // rows per chunk
constexpr int kBox = 16;      // rows per TMA box (and per MMA tile)
constexpr int kU = 2;         // consumer warps per group, one tile each
static_assert(kU == 2, "the partial-output exchange pairs two warps");
constexpr int kMaxGroups = 4;
constexpr int kMaxStages = 4; // per group
constexpr int kQPitch = 272;  // bytes per staged query row (256 + 16 padding)
constexpr int kMaxRowsChunk = 1024;

// Chunk header words.
enum : int {
  H_JOB = 0,    // launch-local job index
  H_BASE,       // job row of stage row 0
  H_VALID,      // live rows of the chunk (stage rows [0, valid)), new row included
  H_LOADED,     // rows with copied old scores / positions
  H_FLAGS,
  H_NEWROW,     // stage row of the new row (if F_NEW)
  H_T,          // position of the new row
  H_NTOT,       // rows of the job with the new row
  H_NA,         // rows of segment A
  H_WORDS = 16
};
enum : int { F_FIRST = 1, F_LAST = 2, F_NEW = 4, F_SKIP = 8 };

// Byte offsets inside one stage.
struct ChunkStage {
  static constexpr uint32_t k0 = 0, k1 = kCR * 128, v0 = 2 * kCR * 128,
                            v1 = 3 * kCR * 128, q = 4 * kCR * 128,
                            kn = q + 8 * kQPitch, vn = kn + 256, sc = vn + 256,
                            ps = sc + 4 * kCR, hdr = ps + 4 * kCR,
                            bytes = ((hdr + 4 * H_WORDS) + 1023) / 1024 * 1024;
};

// Byte offsets inside one group's area (after the rings).
struct ChunkGroup {
  uint32_t xs, ox, lg, sc, ps, ns, bytes;
  __host__ __device__ explicit ChunkGroup(int n_max) {
    const int n = round_up16(n_max);
    xs = 0;                      // [kU][5] 16-byte slots
    ox = 256;                    // [kU][4][32] float4 partial outputs: the
                                 // 4 head-dim tiles the other warp owns
    lg = ox + kU * 4 * 32 * 16;  // [n][8] scaled logits
    sc = lg + n * 8 * 4;         // [n] old scores
    ps = sc + n * 4;             // [n] positions
    ns = ps + n * 4;             // [n] new scores
    bytes = ((ns + n * 4) + 127) / 128 * 128;
  }
};

struct Job {
  size_t ug;    // cache unit (the parent's, for candidates)
  size_t orow;  // row of the job in q / k_new / v_new / out
  size_t cu;    // candidate unit (candidates only)
};

__device__ __forceinline__ Job job_of(const ChunkParams &p, int idx) {
  const int per = p.c.S * p.nl * p.c.H;  // units of the call
  const int cand = idx / per, r = idx % per;
  const int h = r % p.c.H, lr = (r / p.c.H) % p.nl, sq = r / (p.c.H * p.nl);
  Job j;
  j.ug = ((size_t)sq * p.c.L + p.lb + lr) * p.c.H + h;
  j.orow = (size_t)cand * per + ((size_t)sq * p.nl + lr) * p.c.H + h;
  j.cu = (size_t)cand * ((size_t)p.c.S * p.c.L * p.c.H) + j.ug;
  return j;
}

__device__ __forceinline__ void group_bar(int id, int threads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

// Producer warp of one group: every chunk of the group's jobs, in order.
template <bool kFork>
__device__ void produce(const ChunkParams &p, const CUtensorMap *tmK,
                        const CUtensorMap *tmV, const CUtensorMap *tmTK,
                        const CUtensorMap *tmTV, unsigned char *ring,
                        uint64_t *full, uint64_t *empty, int g, int mine,
                        int lane, volatile int *abort, int *issued) {
  const CacheView &c = p.c;
  // Test hook: group 0 of CTA 0 never loads its first job (no copy is
  // issued, so there is nothing to drain); its consumers' wait runs out.
  if (c.hold_first && blockIdx.x == 0 && g == 0) return;
  int seq = 0;
  for (int k = g; k < mine; k += p.n_groups) {
    const int idx = (int)blockIdx.x + k * (int)gridDim.x;
    const Job jb = job_of(p, idx);
    int nA, nB, t;
    bool ok;
    if (kFork) {
      nA = c.state[4 * jb.ug];
      nB = p.f.tlen[jb.cu];
      t = c.state[4 * jb.ug + 1] + nB;
      ok = nA >= 0 && nB >= 0 && nB + 1 <= p.f.tcap && nA + nB + 1 <= p.n_max;
    } else {
      nA = 0;
      nB = c.state[4 * jb.ug];
      t = c.state[4 * jb.ug + 1];
      ok = nB >= 0 && nB + 1 <= c.cap && nB + 1 <= p.n_max;
    }
    if (!ok && lane == 0) atomicOr(c.err, kFork ? ERR_CAPACITY : ERR_LENGTH);
    const int cA = ok ? (nA + kCR - 1) / kCR : 0;
    const int total = ok ? cA + nB / kCR + 1 : 1;
    for (int ci = 0; ci < total; ++ci, ++seq) {
      const int s = seq % p.n_stages;
      const uint32_t ph = (uint32_t)(seq / p.n_stages) & 1u;
      int got = 1;
      if (lane == 0)
        got = mbar_wait(smem_u32(&empty[s]), ph ^ 1u, abort, c.wait_ns);
      got = __shfl_sync(0xffffffffu, got, 0);
      if (!got) {
        if (lane == 0) {
          atomicOr(c.err, ERR_TIMEOUT);
          *abort = 1;
        }
        return;
      }
      __syncwarp();
      unsigned char *st = ring + s * ChunkStage::bytes;
      const uint32_t s0 = smem_u32(st);
      const uint32_t bar = smem_u32(&full[s]);
      const bool segA = ci < cA;
      const int first = 32 * (segA ? ci : ci - cA);  // row within the segment
      const int nseg = segA ? nA : nB;
      const int loaded = ok ? max(0, min(kCR, nseg - first)) : 0;
      const bool has_new = ok && !segA && nB - first < kCR;
      const int boxes = (loaded + kBox - 1) / kBox;
      if (lane == 0) {
        int *h = reinterpret_cast<int *>(st + ChunkStage::hdr);
        h[H_JOB] = idx;
        h[H_BASE] = (segA ? 0 : nA) + first;
        h[H_VALID] = loaded + (has_new ? 1 : 0);
        h[H_LOADED] = loaded;
        h[H_FLAGS] = (ci == 0 ? F_FIRST : 0) | (ci == total - 1 ? F_LAST : 0) |
                     (has_new ? F_NEW : 0) | (ok ? 0 : F_SKIP);
        h[H_NEWROW] = nB - first;
        h[H_T] = t;
        h[H_NTOT] = nA + nB + 1;
        h[H_NA] = nA;
        mbar_expect_tx(bar, (uint32_t)boxes * 4u * kBox * 128u);
        const CUtensorMap *mk = (kFork && !segA) ? tmTK : tmK;
        const CUtensorMap *mv = (kFork && !segA) ? tmTV : tmV;
        const size_t y0 = (kFork && !segA) ? jb.cu * (size_t)p.f.tcap
                                           : jb.ug * (size_t)c.cap;
        for (int bx = 0; bx < boxes; ++bx) {
          const int y = (int)(y0 + first + bx * kBox);
          const uint32_t off = bx * kBox * 128;
          tma_load_2d(s0 + ChunkStage::k0 + off, mk, 0, y, bar);
          tma_load_2d(s0 + ChunkStage::k1 + off, mk, 64, y, bar);
          tma_load_2d(s0 + ChunkStage::v0 + off, mv, 0, y, bar);
          tma_load_2d(s0 + ChunkStage::v1 + off, mv, 64, y, bar);
        }
      }
      if (ok) {
        if (ci == 0) {  // the job's query rows
          const unsigned char *q = reinterpret_cast<const unsigned char *>(
              p.q + jb.orow * c.G * 128);
          for (int i = lane; i < c.G * 16; i += 32)
            cp_async16(s0 + ChunkStage::q + (i >> 4) * kQPitch + (i & 15) * 16,
                       q + i * 16);
        }
        if (has_new)
          cp_async16(s0 + (lane < 16 ? ChunkStage::kn : ChunkStage::vn) +
                         (lane & 15) * 16,
                     reinterpret_cast<const unsigned char *>(
                         (lane < 16 ? p.k_new : p.v_new) + jb.orow * 128) +
                         (lane & 15) * 16);
        // Old scores (and positions) of the loaded rows, in 16-byte pieces
        // (rows are padded to a multiple of 16 in every score array).
        const float *sc;
        const int32_t *ps = nullptr;
        if (kFork)
          sc = segA ? p.f.pscore + jb.cu * c.sstride
                    : p.f.tscore + jb.cu * p.f.tstride;
        else {
          sc = c.score + jb.ug * c.sstride;
          ps = c.pos + jb.ug * c.sstride;
        }
        const int pieces = (loaded + 3) / 4;
        if (lane < pieces)
          cp_async16(s0 + ChunkStage::sc + lane * 16, sc + first + 4 * lane);
        else if (!kFork && lane >= 16 && lane - 16 < pieces)
          cp_async16(s0 + ChunkStage::ps + (lane - 16) * 16,
                     ps + first + 4 * (lane - 16));
      }
      cp_async_arrive_noinc(bar);
      if (lane == 0) *issued = seq + 1;
    }
  }
}

template <bool kFork, bool kOutBf16>
__global__ void __launch_bounds__(kMaxGroups * (kU + 1) * 32, 1)
    chunk_step_kernel(const __grid_constant__ CUtensorMap tmK,
                      const __grid_constant__ CUtensorMap tmV,
                      const __grid_constant__ CUtensorMap tmTK,
                      const __grid_constant__ CUtensorMap tmTV,
                      const ChunkParams p) {
  extern __shared__ unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kMaxGroups][kMaxStages];
  __shared__ __align__(8) uint64_t empty_bar[kMaxGroups][kMaxStages];
  __shared__ int issued_n[kMaxGroups], consumed_n[kMaxGroups];
  __shared__ volatile int s_abort;
  __shared__ volatile int s_ok[kMaxGroups];
  unsigned char *smem = reinterpret_cast<unsigned char *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const CacheView &c = p.c;
  const int G = c.G;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_jobs = p.n_jobs;
  const int mine = (int)blockIdx.x < n_jobs
                       ? (n_jobs - 1 - (int)blockIdx.x) / (int)gridDim.x + 1
                       : 0;
  const int consumers = p.n_groups * kU;
  const ChunkGroup GL(p.n_max);
  const uint32_t ring_bytes = p.n_stages * ChunkStage::bytes;

  if (threadIdx.x == 0) {
    prefetch_tmap(&tmK);
    prefetch_tmap(&tmV);
    if (kFork) {
      prefetch_tmap(&tmTK);
      prefetch_tmap(&tmTV);
    }
    for (int g = 0; g < p.n_groups; ++g) {
      for (int s = 0; s < p.n_stages; ++s) {
        mbar_init(smem_u32(&full_bar[g][s]), 1 + 32);  // TMA + producer lanes
        mbar_init(smem_u32(&empty_bar[g][s]), kU);
      }
      issued_n[g] = 0;
      consumed_n[g] = 0;
    }
    s_abort = 0;
    fence_mbar_init();
  }
  // Query rows of heads >= G are never copied: zero them once per stage.
  for (int i = threadIdx.x; i < p.n_groups * p.n_stages * 8 * (kQPitch / 16);
       i += blockDim.x) {
    const int st = i / (8 * (kQPitch / 16)), r = i % (8 * (kQPitch / 16));
    const int g = st / p.n_stages, s = st % p.n_stages;
    if (r >= G * (kQPitch / 16))
      reinterpret_cast<int4 *>(smem + g * ring_bytes + s * ChunkStage::bytes +
                               ChunkStage::q)[r] = make_int4(0, 0, 0, 0);
  }
  fence_proxy_async();
  __syncthreads();
  pdl_begin();

  if (warp >= consumers) {
    const int g = warp - consumers;
    if (g < p.n_groups)
      produce<kFork>(p, &tmK, &tmV, &tmTK, &tmTV, smem + g * ring_bytes,
                     full_bar[g], empty_bar[g], g, mine, lane, &s_abort,
                     &issued_n[g]);
  } else {
    const int g = warp / kU, w = warp % kU, bar_id = 1 + g;
    unsigned char *ring = smem + g * ring_bytes;
    unsigned char *ga =
        smem + p.n_groups * ring_bytes + g * GL.bytes;
    float *LG = reinterpret_cast<float *>(ga + GL.lg);
    float *GSC = reinterpret_cast<float *>(ga + GL.sc);
    int32_t *GPS = reinterpret_cast<int32_t *>(ga + GL.ps);
    float *GNS = reinterpret_cast<float *>(ga + GL.ns);
    float4 *XS4 = reinterpret_cast<float4 *>(ga + GL.xs);
    float4 *OX = reinterpret_cast<float4 *>(ga + GL.ox);
    const int r0l = lane >> 2, c2 = (lane & 3) * 2;
    int seq = 0;
    bool stop = false;
    for (int k = g; k < mine && !stop; k += p.n_groups) {
      float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
      float o[8][4];
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
      uint32_t qb[8][2];
      int idx = 0, t = 0, ntot = 0, nA = 0;
      int4 nrow = make_int4(0, 0, 0, 0);  // warp 0: the new k (lanes 0-15) / v row
      bool skip = false;
      for (;;) {
        const int s = seq % p.n_stages;
        const uint32_t ph = (uint32_t)(seq / p.n_stages) & 1u;
        // One warp waits (bounded) and tells the group, so that both warps
        // take the same branch before the group's next barrier.
        if (w == 0 && lane == 0) {
          const bool ok =
              mbar_wait(smem_u32(&full_bar[g][s]), ph, &s_abort, c.wait_ns);
          s_ok[g] = ok ? 1 : 0;
          if (!ok) {
            atomicOr(c.err, ERR_TIMEOUT);
            s_abort = 1;
          }
        }
        group_bar(bar_id, 32 * kU);
        if (!s_ok[g]) {
          stop = true;
          break;
        }
        mbar_try_wait(smem_u32(&full_bar[g][s]), ph);  // acquire for this thread
        unsigned char *st = ring + s * ChunkStage::bytes;
        const int *h = reinterpret_cast<const int *>(st + ChunkStage::hdr);
        const int flags = h[H_FLAGS], base = h[H_BASE], valid = h[H_VALID];
        const int loaded = h[H_LOADED];
        if (flags & F_FIRST) {
          idx = h[H_JOB];
          t = h[H_T];
          ntot = h[H_NTOT];
          nA = h[H_NA];
          const uint32_t qa = smem_u32(st + ChunkStage::q) +
                              (lane & 7) * kQPitch + (lane >> 3) * 16;
#pragma unroll
          for (int i = 0; i < 4; ++i)
            ldsm_x4(qa + i * 64, qb[2 * i][0], qb[2 * i][1], qb[2 * i + 1][0],
                    qb[2 * i + 1][1]);
        }
        skip = (flags & F_SKIP) != 0;
        unsigned char *K0 = st + ChunkStage::k0, *K1 = st + ChunkStage::k1;
        unsigned char *V0 = st + ChunkStage::v0, *V1 = st + ChunkStage::v1;
        const int tr0 = kBox * w;
        bool wrote = false;  // generic-proxy writes to the stage
        if (!skip && (flags & F_NEW) && w == 0)
          nrow = *reinterpret_cast<const int4 *>(
              st + (lane < 16 ? ChunkStage::kn : ChunkStage::vn) + (lane & 15) * 16);
        if (!skip && tr0 < valid) {
          // New row (from the inputs) and zero V past the live rows.
          if ((flags & F_NEW) && h[H_NEWROW] >= tr0 && h[H_NEWROW] < tr0 + kBox) {
            const int rn = h[H_NEWROW];
            const int ch = lane & 15, half = ch >> 3, cc = ch & 7;
            unsigned char *dst = lane < 16 ? (half ? K1 : K0) : (half ? V1 : V0);
            const unsigned char *src = st + (lane < 16 ? ChunkStage::kn : ChunkStage::vn);
            *reinterpret_cast<int4 *>(dst + rn * 128 + ((cc ^ (rn & 7)) << 4)) =
                *reinterpret_cast<const int4 *>(src + ch * 16);
            wrote = true;
          }
          wrote = wrote || valid < tr0 + kBox;
          for (int i = lane; i < (tr0 + kBox - max(tr0, valid)) * 16; i += 32) {
            const int r = max(tr0, valid) + (i >> 4), c16 = i & 15;
            *reinterpret_cast<int4 *>((c16 < 8 ? V0 : V1) + r * 128 +
                                      (c16 & 7) * 16) = make_int4(0, 0, 0, 0);
          }
          // Old scores / positions of this tile's rows into the group area.
          if (lane < kBox) {
            const int r = tr0 + lane;
            if (r < loaded) {
              GSC[base + r] = reinterpret_cast<const float *>(st + ChunkStage::sc)[r];
              GPS[base + r] = reinterpret_cast<const int32_t *>(st + ChunkStage::ps)[r];
            } else if (r < valid) {  // the new row
              GSC[base + r] = 0.f;
              GPS[base + r] = t;
            }
          }
          __syncwarp();
          float sa[4] = {0.f, 0.f, 0.f, 0.f}, sb[4] = {0.f, 0.f, 0.f, 0.f};
          {
            const int row = tr0 + (lane & 7) + ((lane >> 3) & 1) * 8;
            const uint32_t b0 = smem_u32(K0) + row * 128, b1 = smem_u32(K1) + row * 128;
#pragma unroll
            for (int ks = 0; ks < 8; ++ks) {
              const int cc = ((ks & 3) << 1) + (lane >> 4);
              const uint32_t addr = (ks >> 2 ? b1 : b0) + ((cc ^ (row & 7)) << 4);
              uint32_t a0, a1, a2, a3;
              ldsm_x4(addr, a0, a1, a2, a3);
              if (ks & 1) mma_bf16(sb, a0, a1, a2, a3, qb[ks][0], qb[ks][1]);
              else mma_bf16(sa, a0, a1, a2, a3, qb[ks][0], qb[ks][1]);
            }
          }
          const int ra = tr0 + r0l, rb = ra + 8;  // stage rows
          float s4[4];
          s4[0] = ra < valid ? (sa[0] + sb[0]) * p.scale_log2e : -INFINITY;
          s4[1] = ra < valid ? (sa[1] + sb[1]) * p.scale_log2e : -INFINITY;
          s4[2] = rb < valid ? (sa[2] + sb[2]) * p.scale_log2e : -INFINITY;
          s4[3] = rb < valid ? (sa[3] + sb[3]) * p.scale_log2e : -INFINITY;
          if (ra < valid)
            *reinterpret_cast<float2 *>(LG + (base + ra) * 8 + c2) =
                make_float2(s4[0], s4[1]);
          if (rb < valid)
            *reinterpret_cast<float2 *>(LG + (base + rb) * 8 + c2) =
                make_float2(s4[2], s4[3]);
          float x0 = fmaxf(s4[0], s4[2]), x1 = fmaxf(s4[1], s4[3]);
#pragma unroll
          for (int off = 4; off < 32; off <<= 1) {
            x0 = fmaxf(x0, __shfl_xor_sync(0xffffffffu, x0, off));
            x1 = fmaxf(x1, __shfl_xor_sync(0xffffffffu, x1, off));
          }
          // Row tr0 is live, so the new maxima are finite.
          const float n0 = fmaxf(m0, x0), n1 = fmaxf(m1, x1);
          const float a0 = ex2(m0 - n0), a1 = ex2(m1 - n1);
          m0 = n0;
          m1 = n1;
          s4[0] = ex2(s4[0] - m0);
          s4[1] = ex2(s4[1] - m1);
          s4[2] = ex2(s4[2] - m0);
          s4[3] = ex2(s4[3] - m1);
          l0 = l0 * a0 + s4[0] + s4[2];
          l1 = l1 * a1 + s4[1] + s4[3];
          {
            const uint64_t a2 = pk2(a0, a1);  // (head c2, head c2 + 1)
#pragma unroll
            for (int mt = 0; mt < 8; ++mt) {
              upk2(mul2(pk2(o[mt][0], o[mt][1]), a2), o[mt][0], o[mt][1]);
              upk2(mul2(pk2(o[mt][2], o[mt][3]), a2), o[mt][2], o[mt][3]);
            }
          }
          const uint32_t h0 = pack_bf16(s4[0], s4[1]), h1 = pack_bf16(s4[2], s4[3]);
          const __nv_bfloat162 hb0 = *reinterpret_cast<const __nv_bfloat162 *>(&h0);
          const __nv_bfloat162 hb1 = *reinterpret_cast<const __nv_bfloat162 *>(&h1);
          const uint32_t bp0 = movm_t(h0), bp1 = movm_t(h1);
          const uint32_t bl0 = movm_t(pack_bf16(s4[0] - __low2float(hb0), s4[1] - __high2float(hb0)));
          const uint32_t bl1 = movm_t(pack_bf16(s4[2] - __low2float(hb1), s4[3] - __high2float(hb1)));
          const int row = tr0 + (lane & 7) + ((lane >> 4) << 3);
          const uint32_t b0 = smem_u32(V0) + row * 128, b1 = smem_u32(V1) + row * 128;
#pragma unroll
          for (int mt = 0; mt < 8; ++mt) {
            const int c16 = 2 * mt + ((lane >> 3) & 1);
            const uint32_t addr = (c16 >> 3 ? b1 : b0) + (((c16 & 7) ^ (row & 7)) << 4);
            uint32_t v0, v1, v2, v3;
            ldsm_x4_t(addr, v0, v1, v2, v3);
            mma_bf16(o[mt], v0, v1, v2, v3, bp0, bp1);
            mma_bf16(o[mt], v0, v1, v2, v3, bl0, bl1);
          }
        }
        // Release the stage (the fence orders this warp's writes to it, if
        // any, before the next TMA refill).
        if (wrote) fence_proxy_async();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(smem_u32(&empty_bar[g][s]));
          if (w == 0) consumed_n[g] = seq + 1;
        }
        ++seq;
        if (flags & F_LAST) break;
      }
      if (stop || skip) continue;

      // ---- the job's back part: merge, output, scores, eviction ----
#pragma unroll
      for (int off = 4; off < 32; off <<= 1) {
        l0 += __shfl_xor_sync(0xffffffffu, l0, off);
        l1 += __shfl_xor_sync(0xffffffffu, l1, off);
      }
      if (lane < 4) XS4[w * 5 + lane] = make_float4(m0, m1, l0, l1);
      // The partials of the head-dim tiles the other warp owns (mt of the
      // other parity); each warp keeps its own tiles' partials in registers.
#pragma unroll
      for (int mt = 0; mt < 8; ++mt)
        if ((mt & 1) != w)
          OX[(w * 4 + (mt >> 1)) * 32 + lane] =
              make_float4(o[mt][0], o[mt][1], o[mt][2], o[mt][3]);
      group_bar(bar_id, 32 * kU);
      // Per head: the merged maximum and 1 / sum, for all 8 heads (the
      // scores need every head) and the warps' rescale factors for this
      // lane's heads c2, c2 + 1.
      float Mh[8], iZ[8], fv0[kU], fv1[kU];
#pragma unroll
      for (int cp = 0; cp < 4; ++cp) {
        float4 r[kU];
        float Ma = -INFINITY, Mb = -INFINITY;
#pragma unroll
        for (int v = 0; v < kU; ++v) {
          r[v] = XS4[v * 5 + cp];
          if (r[v].z > 0.f) Ma = fmaxf(Ma, r[v].x);
          if (r[v].w > 0.f) Mb = fmaxf(Mb, r[v].y);
        }
        float Za = 0.f, Zb = 0.f, ea[kU], eb[kU];
#pragma unroll
        for (int v = 0; v < kU; ++v) {
          ea[v] = r[v].z > 0.f ? ex2(r[v].x - Ma) : 0.f;
          eb[v] = r[v].w > 0.f ? ex2(r[v].y - Mb) : 0.f;
          Za += r[v].z * ea[v];
          Zb += r[v].w * eb[v];
        }
        const float ia = rcp(Za), ib = rcp(Zb);
        Mh[2 * cp] = Ma;
        Mh[2 * cp + 1] = Mb;
        iZ[2 * cp] = ia;
        iZ[2 * cp + 1] = ib;
        if (cp == (lane & 3)) {
#pragma unroll
          for (int v = 0; v < kU; ++v) {
            fv0[v] = ea[v] * ia;
            fv1[v] = eb[v] * ib;
          }
        }
        if (w == 0 && lane == 0 &&
            !(Za > 0.5f && Za < INFINITY && Zb > 0.5f && Zb < INFINITY))
          atomicOr(c.err, ERR_NONFINITE);
      }
      const Job jb = job_of(p, idx);
      // Output: warp w owns head-dim tiles of parity w; the two warps'
      // terms are added in warp order.
      {
        constexpr int osz = kOutBf16 ? 2 : 4;
        unsigned char *gout = reinterpret_cast<unsigned char *>(p.out) +
                              jb.orow * G * 128 * osz;
#pragma unroll
        for (int mt = 0; mt < 8; ++mt) {
          if ((mt & 1) != w) continue;
          const float4 mine = make_float4(o[mt][0], o[mt][1], o[mt][2], o[mt][3]);
          const float4 other = OX[((1 - w) * 4 + (mt >> 1)) * 32 + lane];
          float e0 = 0.f, e1 = 0.f, e2 = 0.f, e3 = 0.f;
#pragma unroll
          for (int v = 0; v < kU; ++v) {
            const float4 x = v == w ? mine : other;
            e0 += x.x * fv0[v];
            e1 += x.y * fv1[v];
            e2 += x.z * fv0[v];
            e3 += x.w * fv1[v];
          }
          if (kOutBf16) {
            const uint32_t lo = movm_t(pack_bf16(e0, e1));
            const uint32_t hi = movm_t(pack_bf16(e2, e3));
            const int gg = lane >> 2, dd = 16 * mt + 2 * (lane & 3);
            if (gg < G) {
              *reinterpret_cast<uint32_t *>(gout + ((size_t)gg * 128 + dd) * 2) = lo;
              *reinterpret_cast<uint32_t *>(gout + ((size_t)gg * 128 + dd + 8) * 2) = hi;
            }
          } else {
            float *of = reinterpret_cast<float *>(gout);
            const int d0 = 16 * mt + r0l;
            if (c2 < G) {
              of[c2 * 128 + d0] = e0;
              of[c2 * 128 + d0 + 8] = e2;
            }
            if (c2 + 1 < G) {
              of[(c2 + 1) * 128 + d0] = e1;
              of[(c2 + 1) * 128 + d0 + 8] = e3;
            }
          }
        }
      }
      // Accumulated attention of every row from the kept logits; the
      // eviction candidate (lowest (score, -position) outside the window).
      const int tid = w * 32 + lane;
      const int wlo = t - p.window;
      const bool evict = !kFork && p.evict && ntot > p.budget + p.window;
      unsigned long long best = ~0ull;
      int bi = -1;
      for (int r = tid; r < ntot; r += 32 * kU) {
        const float4 la = *reinterpret_cast<const float4 *>(LG + r * 8);
        const float4 lb = *reinterpret_cast<const float4 *>(LG + r * 8 + 4);
        const float lg8[8] = {la.x, la.y, la.z, la.w, lb.x, lb.y, lb.z, lb.w};
        float acc = 0.f;
#pragma unroll
        for (int gg = 0; gg < 8; ++gg)
          if (gg < G) acc += ex2(lg8[gg] - Mh[gg]) * iZ[gg];
        const float sc = GSC[r] + acc * p.inv_g;
        GNS[r] = sc;
        if (evict) {
          const int pr = GPS[r];
          if (pr <= wlo) {
            const unsigned long long key =
                ((unsigned long long)__float_as_uint(sc) << 32) |
                (unsigned long long)(0xFFFFFFFFu - (unsigned)pr);
            if (key < best) {
              best = key;
              bi = r;
            }
          }
        }
      }
      int victim = -1;
      if (evict) {
#pragma unroll
        for (int o2 = 16; o2 > 0; o2 >>= 1) {
          const unsigned long long ob = __shfl_xor_sync(0xffffffffu, best, o2);
          const int oi = __shfl_xor_sync(0xffffffffu, bi, o2);
          if (ob < best) {
            best = ob;
            bi = oi;
          }
        }
        uint4 *XW = reinterpret_cast<uint4 *>(XS4);
        if (lane == 0)
          XW[w * 5 + 4] = make_uint4((uint32_t)best, (uint32_t)(best >> 32),
                                     (uint32_t)bi, 0u);
      }
      group_bar(bar_id, 32 * kU);  // new scores (and candidates) visible
      if (evict) {
        const uint4 *XW = reinterpret_cast<const uint4 *>(XS4);
#pragma unroll
        for (int v = 0; v < kU; ++v) {
          const uint4 a = XW[v * 5 + 4];
          const unsigned long long kb = ((unsigned long long)a.y << 32) | a.x;
          if (kb < best) {
            best = kb;
            bi = (int)a.z;
          }
        }
        victim = bi;
      }
      // Write back.
      if (kFork) {
        const int nt = ntot - 1 - nA;  // tail rows before the append
        float *ps = p.f.pscore + jb.cu * c.sstride;
        float *ts = p.f.tscore + jb.cu * p.f.tstride;
        for (int r = tid; r < ntot; r += 32 * kU) {
          if (r < nA) ps[r] = GNS[r];
          else ts[r - nA] = GNS[r];
        }
        if (w == 0) {
          __nv_bfloat16 *dst =
              reinterpret_cast<__nv_bfloat16 *>(lane < 16 ? p.f.TK : p.f.TV) +
              (jb.cu * (size_t)p.f.tcap + nt) * 128;
          reinterpret_cast<int4 *>(dst)[lane & 15] = nrow;
          if (lane == 0) {
            p.f.tpos[jb.cu * p.f.tstride + nt] = t;
            p.f.tlen[jb.cu] = nt + 1;
          }
        }
      } else {
        const int m = ntot - 1;  // live rows before the append
        float *gsc = c.score + jb.ug * c.sstride;
        for (int r = tid; r < m; r += 32 * kU)
          gsc[r] = r == victim ? GNS[m] : GNS[r];
        const int slot = victim < 0 ? m : (victim < m ? victim : -1);
        if (w == 0) {
          if (slot >= 0) {
            __nv_bfloat16 *dst =
                reinterpret_cast<__nv_bfloat16 *>(lane < 16 ? c.K : c.V) +
                (jb.ug * (size_t)c.cap + slot) * 128;
            reinterpret_cast<int4 *>(dst)[lane & 15] = nrow;
            if (lane == 0) {
              c.pos[jb.ug * c.sstride + slot] = t;
              if (slot == m) gsc[m] = GNS[m];
            }
          }
          if (lane == 0) {
            c.state[4 * jb.ug] = victim < 0 ? m + 1 : m;
            c.state[4 * jb.ug + 1] = t + 1;
            c.state[4 * jb.ug + 2] = 0;  // R-KV key sum no longer valid
          }
        }
      }
      group_bar(bar_id, 32 * kU);  // the group area is free for the next job
    }
  }
  __syncthreads();
  // After an abort, wait (bounded) for copies still landing in the rings.
  if (s_abort && threadIdx.x == 0) {
    volatile int never = 0;
    for (int g = 0; g < p.n_groups; ++g)
      for (int q = consumed_n[g]; q < issued_n[g]; ++q)
        mbar_wait(smem_u32(&full_bar[g][q % p.n_stages]),
                  (uint32_t)(q / p.n_stages) & 1u, &never);
  }
}

template <bool kFork>
cudaError_t launch_k(const CUtensorMap &tmK, const CUtensorMap &tmV,
                     const CUtensorMap &tmTK, const CUtensorMap &tmTV,
                     const ChunkParams &p, int grid, size_t smem,
                     cudaStream_t st) {
  auto kern = p.c.out_bf16 ? chunk_step_kernel<kFork, true>
                           : chunk_step_kernel<kFork, false>;
  cudaError_t e = cudaFuncSetAttribute(
      kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(kern, dim3(grid), dim3(32 * p.n_groups * (kU + 1)), smem,
                    st, tmK, tmV, tmTK, tmTV, p);
}

}  // namespace

int chunk_box_rows() { return kBox; }
int chunk_max_rows() { return kMaxRowsChunk; }
int chunk_max_groups() { return kMaxGroups; }
int chunk_max_stages() { return kMaxStages; }
size_t chunk_smem_bytes(int n_max, int n_groups, int n_stages) {
  return (size_t)n_groups *
             ((size_t)n_stages * ChunkStage::bytes + ChunkGroup(n_max).bytes) +
         1024;
}

cudaError_t launch_chunk_step(const CUtensorMap &tmK, const CUtensorMap &tmV,
                              const CUtensorMap *tmTK, const CUtensorMap *tmTV,
                              const ChunkParams &p, int grid,
                              cudaStream_t st) {
  if (p.n_groups < 1 || p.n_groups > kMaxGroups || p.n_stages < 2 ||
      p.n_stages > kMaxStages || p.n_max < 1 || p.n_max > kMaxRowsChunk ||
      p.c.G > 8 || (p.fork && (!tmTK || !tmTV)))
    return cudaErrorInvalidValue;
  const size_t smem = chunk_smem_bytes(p.n_max, p.n_groups, p.n_stages);
  if (p.fork)
    return launch_k<true>(tmK, tmV, *tmTK, *tmTV, p, grid, smem, st);
  return launch_k<false>(tmK, tmV, tmK, tmV, p, grid, smem, st);
}

}  // namespace kvr
