// kvr_fork_batch.cu -- the candidate-batched decode step of stepwise best-of-N
// (Sec. 2.2 Eq. 2, App. C): N candidates share the parent's live rows as
// a read-only prefix and each has a private tail.  Per candidate: append +
// Attn(q_t, C) (Eq. 1) over prefix + tail + new row, the candidate's
// accumulated attention (Sec. 2.1, mean over the G heads) of every row, and
// the new row appended to the tail (eviction is deferred to the commit).
// bf16, head_dim 128, G <= 8, N <= 8.
//
// Design (GB300, sm_103a):
//  - Persistent CTAs, one per SM, each working through units (sequence,
//    layer, KV head).  One warp per candidate plus a producer warp.
//  - A two-stage ring of 64 KB blocks: a prefix block holds up to 128 of the
//    parent's rows and serves all N candidates, so each prefix row crosses
//    HBM once per unit; a tail block holds T = 16 * (8 / N) rows of every
//    candidate's tail side by side.  A full prefix block is one 128-row
//    128B-swizzled TMA box per quarter (K columns 0-63 and 64-127, V
//    likewise), a partial one 16-row boxes; a tail block is one box per
//    quarter of a 3-D tensor map whose outer dimension is the candidate.  So
//    a block costs the TMA unit 4 to 32 instructions rather than 4 per
//    candidate and box: the instruction issue rate, not HBM, limited a first
//    version with per-candidate boxes.  The producer lanes fetch the new k/v
//    rows and the old scores with cp.async onto the block's mbarrier, and
//    lane 0 writes a block header.  Each warp loads its candidate's query
//    rows straight into MMA fragments one unit ahead, so they take no ring
//    space.
//  - Each warp runs its candidate's online softmax over the unit's blocks,
//    up to four 16-row tiles per update (QK^T of the group, one rescale,
//    then PV; bf16 mma.sync, P split hi + lo), and keeps the scaled logits
//    and old scores of every row in its own area, so the score update uses
//    exact probabilities at the end, with no cross-warp merge.
//  - Rows past the live ones in a loaded box are masked: logits by select,
//    V by zeroing the affected halves of the ldmatrix fragments, so a shared
//    block is never written (the new row is inserted only into the owning
//    candidate's slice).
//  - Launched with programmatic stream serialization; every mbarrier wait is
//    bounded (about 2 s) and on timeout sets ERR_TIMEOUT and drains its copies.
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

constexpr int kBox = 16;         // rows per partial-prefix TMA box, per MMA tile
constexpr int kBlockRows = 128;  // rows of a block
constexpr int kMaxCand = 8;
constexpr int kStages = 2;
constexpr int kGroupTiles = 4;   // tiles per online-softmax update

enum : int {
  H_JOB = 0,  // launch-local unit index
  H_FIRST,    // first row of the block within its segment
  H_ROWS,     // loaded rows (prefix: of the block; tail: per candidate)
  H_FLAGS,
  H_NP,       // prefix rows
  H_NT,       // tail rows before the append
  H_T,        // position of the new row
  H_WORDS = 16
};
enum : int { F_FIRST = 1, F_LAST = 2, F_NEW = 4, F_SKIP = 8, F_TAIL = 16 };

struct BatchStage {
  static constexpr uint32_t k0 = 0, k1 = kBlockRows * 128,
                            v0 = 2 * kBlockRows * 128,
                            v1 = 3 * kBlockRows * 128,
                            kn = 4 * kBlockRows * 128,              // [c][256]
                            vn = kn + kMaxCand * 256,               // [c][256]
                            sc = vn + kMaxCand * 256,               // [c][128]
                            hdr = sc + kMaxCand * kBlockRows * 4,
                            bytes = ((hdr + 4 * H_WORDS) + 1023) / 1024 * 1024;
};

// Tail rows per candidate in a tail block (N * T <= kBlockRows; a multiple
// of 16, so every candidate's slice starts on a whole tile, 1024-byte
// aligned as the 128B swizzle needs).
__host__ __device__ inline int tail_rows(int N) { return kBox * (8 / N); }
__host__ __device__ inline int warp_area_bytes(int n_max) {
  return round_up16(n_max) * (8 + 1) * 4;  // logits [n][8], old scores [n]
}

__device__ __forceinline__ void group_bar(int id, int threads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

// Zero the halves of a transposed-V A fragment (k index = tile row) whose
// rows are at or past `valid`: a0/a1 hold rows 2t, 2t+1, a2/a3 rows +8.
__device__ __forceinline__ void mask_rows(uint32_t &a0, uint32_t &a1,
                                          uint32_t &a2, uint32_t &a3,
                                          int valid, int lane) {
  const int r = 2 * (lane & 3);
  const uint32_t lo = (r < valid ? 0x0000FFFFu : 0u) | (r + 1 < valid ? 0xFFFF0000u : 0u);
  const uint32_t hi = (r + 8 < valid ? 0x0000FFFFu : 0u) | (r + 9 < valid ? 0xFFFF0000u : 0u);
  a0 &= lo;
  a1 &= lo;
  a2 &= hi;
  a3 &= hi;
}

// Up to kGroupTiles 16-row tiles for one warp, processed together: the
// logits of every tile (stored at LG[(row0 + 16 t + r) * 8 + g]), one online
// softmax update for the group (one maximum, one rescale), then PV over the
// group.  K/V point at the first tile's row in the block's quarters; tile t
// has min(16, rows - 16 t) live rows, the rest masked.
__device__ __forceinline__ void tile_group(const unsigned char *K0,
                                           const unsigned char *K1,
                                           const unsigned char *V0,
                                           const unsigned char *V1, int rows,
                                           const uint32_t (&qb)[8][2],
                                           float scale_log2e, float *LG,
                                           int row0, float &m0, float &m1,
                                           float &l0, float &l1,
                                           float (&o)[8][4], int lane) {
  const int r0l = lane >> 2, c2 = (lane & 3) * 2;
  const int nt = min(kGroupTiles, (rows + kBox - 1) / kBox);
  float s4[kGroupTiles][4];
#pragma unroll
  for (int t = 0; t < kGroupTiles; ++t) {
    float sa[4] = {0.f, 0.f, 0.f, 0.f}, sb[4] = {0.f, 0.f, 0.f, 0.f};
    if (t < nt) {
      const int row = t * kBox + (lane & 7) + ((lane >> 3) & 1) * 8;
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
    const int valid = rows - t * kBox;  // live rows of this tile (if > 0)
    s4[t][0] = r0l < valid ? (sa[0] + sb[0]) * scale_log2e : -INFINITY;
    s4[t][1] = r0l < valid ? (sa[1] + sb[1]) * scale_log2e : -INFINITY;
    s4[t][2] = r0l + 8 < valid ? (sa[2] + sb[2]) * scale_log2e : -INFINITY;
    s4[t][3] = r0l + 8 < valid ? (sa[3] + sb[3]) * scale_log2e : -INFINITY;
    if (r0l < valid)
      *reinterpret_cast<float2 *>(LG + (row0 + t * kBox + r0l) * 8 + c2) =
          make_float2(s4[t][0], s4[t][1]);
    if (r0l + 8 < valid)
      *reinterpret_cast<float2 *>(LG + (row0 + t * kBox + r0l + 8) * 8 + c2) =
          make_float2(s4[t][2], s4[t][3]);
  }
  float x0 = -INFINITY, x1 = -INFINITY;
#pragma unroll
  for (int t = 0; t < kGroupTiles; ++t) {
    x0 = fmaxf(x0, fmaxf(s4[t][0], s4[t][2]));
    x1 = fmaxf(x1, fmaxf(s4[t][1], s4[t][3]));
  }
#pragma unroll
  for (int off = 4; off < 32; off <<= 1) {
    x0 = fmaxf(x0, __shfl_xor_sync(0xffffffffu, x0, off));
    x1 = fmaxf(x1, __shfl_xor_sync(0xffffffffu, x1, off));
  }
  const float n0 = fmaxf(m0, x0), n1 = fmaxf(m1, x1);  // row 0 is live
  const float a0 = ex2(m0 - n0), a1 = ex2(m1 - n1);
  m0 = n0;
  m1 = n1;
  l0 *= a0;
  l1 *= a1;
  {
    const uint64_t a2 = pk2(a0, a1);  // (head c2, head c2 + 1)
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) {
      upk2(mul2(pk2(o[mt][0], o[mt][1]), a2), o[mt][0], o[mt][1]);
      upk2(mul2(pk2(o[mt][2], o[mt][3]), a2), o[mt][2], o[mt][3]);
    }
  }
#pragma unroll
  for (int t = 0; t < kGroupTiles; ++t) {
    if (t >= nt) break;
    const float p0 = ex2(s4[t][0] - m0), p1 = ex2(s4[t][1] - m1);
    const float p2 = ex2(s4[t][2] - m0), p3 = ex2(s4[t][3] - m1);
    l0 += p0 + p2;
    l1 += p1 + p3;
    const uint32_t h0 = pack_bf16(p0, p1), h1 = pack_bf16(p2, p3);
    const __nv_bfloat162 hb0 = *reinterpret_cast<const __nv_bfloat162 *>(&h0);
    const __nv_bfloat162 hb1 = *reinterpret_cast<const __nv_bfloat162 *>(&h1);
    const uint32_t bp0 = movm_t(h0), bp1 = movm_t(h1);
    const uint32_t bl0 = movm_t(pack_bf16(p0 - __low2float(hb0), p1 - __high2float(hb0)));
    const uint32_t bl1 = movm_t(pack_bf16(p2 - __low2float(hb1), p3 - __high2float(hb1)));
    const int valid = rows - t * kBox;
    const int row = t * kBox + (lane & 7) + ((lane >> 4) << 3);
    const uint32_t b0 = smem_u32(V0) + row * 128, b1 = smem_u32(V1) + row * 128;
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) {
      const int c16 = 2 * mt + ((lane >> 3) & 1);
      const uint32_t addr = (c16 >> 3 ? b1 : b0) + (((c16 & 7) ^ (row & 7)) << 4);
      uint32_t v0, v1, v2, v3;
      ldsm_x4_t(addr, v0, v1, v2, v3);
      if (valid < kBox) mask_rows(v0, v1, v2, v3, valid, lane);
      mma_bf16(o[mt], v0, v1, v2, v3, bp0, bp1);
      mma_bf16(o[mt], v0, v1, v2, v3, bl0, bl1);
    }
  }
}

struct Unit {
  size_t ug;    // the parent's unit
  size_t row0;  // unit row of the call ([S][nl][H])
};

__device__ __forceinline__ Unit unit_of(const ForkBatchParams &p, int idx) {
  const CacheView &c = p.f.p;
  const int h = idx % c.H, lr = (idx / c.H) % p.nl, sq = idx / (c.H * p.nl);
  Unit u;
  u.ug = ((size_t)sq * c.L + p.lb + lr) * c.H + h;
  u.row0 = ((size_t)sq * p.nl + lr) * c.H + h;
  return u;
}

__device__ void produce(const ForkBatchParams &p, const CUtensorMap *tmK,
                        const CUtensorMap *tmV, const CUtensorMap *tmK128,
                        const CUtensorMap *tmV128, const CUtensorMap *tmTK,
                        const CUtensorMap *tmTV, unsigned char *ring,
                        uint64_t *full, uint64_t *empty, int mine, int lane,
                        volatile int *abort, int *issued) {
  const ForkView &f = p.f;
  const CacheView &c = f.p;
  const int N = f.N, T = tail_rows(N);
  const size_t units = (size_t)c.S * c.L * c.H;
  const size_t per = (size_t)c.S * p.nl * c.H;  // unit rows of the call
  int seq = 0;
  for (int k = 0; k < mine; ++k) {
    const int idx = (int)blockIdx.x + k * (int)gridDim.x;
    const Unit u = unit_of(p, idx);
    const int np = c.state[4 * u.ug], bp = c.state[4 * u.ug + 1];
    // Every candidate's tail has the same length (one row per call each).
    const int mynt = lane < N ? f.tlen[(size_t)lane * units + u.ug] : -1;
    const int nt = __shfl_sync(0xffffffffu, mynt, 0);
    const bool same = __all_sync(0xffffffffu, lane >= N || mynt == nt);
    const bool ok = same && np >= 0 && nt >= 0 && nt + 1 <= f.tcap &&
                    np + nt + 1 <= p.n_max;
    if (!ok && lane == 0) atomicOr(c.err, same ? ERR_CAPACITY : ERR_LENGTH);
    const int nPB = ok ? (np + kBlockRows - 1) / kBlockRows : 0;
    const int total = ok ? nPB + nt / T + 1 : 1;
    for (int b = 0; b < total; ++b, ++seq) {
      const int s = seq % kStages;
      const uint32_t ph = (uint32_t)(seq / kStages) & 1u;
      int got = 1;
      if (lane == 0) got = mbar_wait(smem_u32(&empty[s]), ph ^ 1u, abort);
      got = __shfl_sync(0xffffffffu, got, 0);
      if (!got) {
        if (lane == 0) {
          atomicOr(c.err, ERR_TIMEOUT);
          *abort = 1;
        }
        return;
      }
      __syncwarp();
      unsigned char *st = ring + s * BatchStage::bytes;
      const uint32_t s0 = smem_u32(st);
      const uint32_t bar = smem_u32(&full[s]);
      const bool tail = b >= nPB;
      const int first = tail ? (b - nPB) * T : b * kBlockRows;
      const int rows = !ok ? 0
                       : tail ? max(0, min(T, nt - first))
                              : min(kBlockRows, np - first);
      const bool has_new = ok && tail && nt - first < T;
      // A tail block is one 3-D box per quarter (T rows x N candidates); a
      // full prefix block one 128-row box; a partial one 16-row boxes.
      const bool full128 = !tail && rows == kBlockRows;
      const int boxes = tail ? (rows > 0 ? 1 : 0)
                             : full128 ? 1 : (rows + kBox - 1) / kBox;
      const uint32_t box_bytes = tail ? (uint32_t)N * T * 128u
                                      : (full128 ? kBlockRows : kBox) * 128u;
      if (lane == 0) {
        int *h = reinterpret_cast<int *>(st + BatchStage::hdr);
        h[H_JOB] = idx;
        h[H_FIRST] = first;
        h[H_ROWS] = rows;
        h[H_FLAGS] = (b == 0 ? F_FIRST : 0) | (b == total - 1 ? F_LAST : 0) |
                     (has_new ? F_NEW : 0) | (ok ? 0 : F_SKIP) |
                     (tail ? F_TAIL : 0);
        h[H_NP] = np;
        h[H_NT] = nt;
        h[H_T] = bp + nt;
        mbar_expect_tx(bar, (uint32_t)boxes * 4u * box_bytes);
      }
      __syncwarp();  // the expected bytes are posted before any copy lands
      if (ok) {
        for (int bx = lane; bx < boxes; bx += 32) {  // one box per lane
          if (tail) {  // rows [first, first + T) of every candidate's tail
            const int y = (int)(u.ug * (size_t)f.tcap + first);
            tma_load_3d(s0 + BatchStage::k0, tmTK, 0, y, 0, bar);
            tma_load_3d(s0 + BatchStage::k1, tmTK, 64, y, 0, bar);
            tma_load_3d(s0 + BatchStage::v0, tmTV, 0, y, 0, bar);
            tma_load_3d(s0 + BatchStage::v1, tmTV, 64, y, 0, bar);
          } else {
            const CUtensorMap *mk = full128 ? tmK128 : tmK;
            const CUtensorMap *mv = full128 ? tmV128 : tmV;
            const int y = (int)(u.ug * (size_t)c.cap + first + bx * kBox);
            const uint32_t off = bx * kBox * 128;
            tma_load_2d(s0 + BatchStage::k0 + off, mk, 0, y, bar);
            tma_load_2d(s0 + BatchStage::k1 + off, mk, 64, y, bar);
            tma_load_2d(s0 + BatchStage::v0 + off, mv, 0, y, bar);
            tma_load_2d(s0 + BatchStage::v1 + off, mv, 64, y, bar);
          }
        }
        if (b == 0) {  // every candidate's new k/v row
          for (int i = lane; i < N * 32; i += 32) {
            const int cand = i >> 5, ch = i & 31;
            const __nv_bfloat16 *src =
                (ch < 16 ? p.k_new : p.v_new) + ((size_t)cand * per + u.row0) * 128;
            cp_async16(s0 + (ch < 16 ? BatchStage::kn : BatchStage::vn) +
                           cand * 256 + (ch & 15) * 16,
                       reinterpret_cast<const unsigned char *>(src) + (ch & 15) * 16);
          }
        }
        // Old scores of the loaded rows, per candidate (rows are padded to a
        // multiple of 16 in every score array).
        const int pieces = (rows + 3) / 4;
        for (int i = lane; i < N * pieces; i += 32) {
          const int cand = i / pieces, pc = i % pieces;
          const size_t cu = (size_t)cand * units + u.ug;
          const float *sc = tail ? f.tscore + cu * f.tstride : f.pscore + cu * c.sstride;
          cp_async16(s0 + BatchStage::sc + (cand * kBlockRows + 4 * pc) * 4,
                     sc + first + 4 * pc);
        }
      }
      cp_async_arrive_noinc(bar);
      if (lane == 0) *issued = seq + 1;
    }
  }
}

template <bool kOutBf16>
__global__ void __launch_bounds__((kMaxCand + 1) * 32, 1)
    fork_batch_kernel(const __grid_constant__ CUtensorMap tmK,
                      const __grid_constant__ CUtensorMap tmV,
                      const __grid_constant__ CUtensorMap tmK128,
                      const __grid_constant__ CUtensorMap tmV128,
                      const __grid_constant__ CUtensorMap tmTK,
                      const __grid_constant__ CUtensorMap tmTV,
                      const ForkBatchParams p) {
  extern __shared__ unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kStages];
  __shared__ __align__(8) uint64_t empty_bar[kStages];
  __shared__ int issued_n, consumed_n;
  __shared__ volatile int s_abort;
  __shared__ volatile int s_ok;
  unsigned char *smem = reinterpret_cast<unsigned char *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const ForkView &f = p.f;
  const CacheView &c = f.p;
  const int G = c.G, N = f.N, T = tail_rows(N);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_units = c.S * p.nl * c.H;
  const int mine = (int)blockIdx.x < n_units
                       ? (n_units - 1 - (int)blockIdx.x) / (int)gridDim.x + 1
                       : 0;
  if (threadIdx.x == 0) {
    prefetch_tmap(&tmK);
    prefetch_tmap(&tmV);
    prefetch_tmap(&tmK128);
    prefetch_tmap(&tmV128);
    prefetch_tmap(&tmTK);
    prefetch_tmap(&tmTV);
    for (int s = 0; s < kStages; ++s) {
      mbar_init(smem_u32(&full_bar[s]), 1 + 32);  // TMA + producer lanes
      mbar_init(smem_u32(&empty_bar[s]), N);      // one arrival per candidate
    }
    issued_n = 0;
    consumed_n = 0;
    s_abort = 0;
    fence_mbar_init();
  }
  __syncthreads();
  pdl_begin();

  if (warp == N) {
    produce(p, &tmK, &tmV, &tmK128, &tmV128, &tmTK, &tmTV, smem, full_bar,
            empty_bar, mine, lane, &s_abort, &issued_n);
  } else if (warp < N) {
    const int cand = warp;
    const size_t units = (size_t)c.S * c.L * c.H;
    const size_t per = (size_t)c.S * p.nl * c.H;
    float *LG = reinterpret_cast<float *>(smem + kStages * BatchStage::bytes +
                                          cand * warp_area_bytes(p.n_max));
    float *GSC = LG + round_up16(p.n_max) * 8;
    const int r0l = lane >> 2, c2 = (lane & 3) * 2;
    // This candidate's query rows of unit k as the QK B operand (lane holds
    // head lane / 4 and the dimension pairs 16 ks + 8 h + 2 (lane % 4)).
    auto load_q = [&](int k, uint32_t (&qb)[8][2]) {
      const Unit u = unit_of(p, (int)blockIdx.x + k * (int)gridDim.x);
      const int g = lane >> 2;
      if (g < G) {
        const uint32_t *q = reinterpret_cast<const uint32_t *>(
                                p.q + (((size_t)cand * per + u.row0) * G + g) * 128) +
                            (lane & 3);
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) {
          qb[ks][0] = __ldg(q + 8 * ks);
          qb[ks][1] = __ldg(q + 8 * ks + 4);
        }
      } else {
#pragma unroll
        for (int ks = 0; ks < 8; ++ks) qb[ks][0] = qb[ks][1] = 0u;
      }
    };
    uint32_t qn[8][2];
    if (mine > 0) load_q(0, qn);
    int seq = 0;
    bool stop = false;
    for (int k = 0; k < mine && !stop; ++k) {
      float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
      float o[8][4];
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
      uint32_t qb[8][2];
#pragma unroll
      for (int ks = 0; ks < 8; ++ks) {
        qb[ks][0] = qn[ks][0];
        qb[ks][1] = qn[ks][1];
      }
      if (k + 1 < mine) load_q(k + 1, qn);  // lands while this unit runs
      int4 nrow = make_int4(0, 0, 0, 0);
      int idx = 0, np = 0, nt = 0, t = 0;
      bool skip = false;
      for (;;) {
        const int s = seq % kStages;
        const uint32_t ph = (uint32_t)(seq / kStages) & 1u;
        // One warp waits (bounded) and tells the others.
        if (warp == 0 && lane == 0) {
          const bool okw = mbar_wait(smem_u32(&full_bar[s]), ph, &s_abort);
          s_ok = okw ? 1 : 0;
          if (!okw) {
            atomicOr(c.err, ERR_TIMEOUT);
            s_abort = 1;
          }
        }
        group_bar(1, 32 * N);
        if (!s_ok) {
          stop = true;
          break;
        }
        mbar_try_wait(smem_u32(&full_bar[s]), ph);  // acquire for this thread
        unsigned char *st = smem + s * BatchStage::bytes;
        const int *h = reinterpret_cast<const int *>(st + BatchStage::hdr);
        const int flags = h[H_FLAGS], first = h[H_FIRST], rows = h[H_ROWS];
        skip = (flags & F_SKIP) != 0;
        bool wrote = false;
        if (!skip) {
          if (flags & F_FIRST) {
            idx = h[H_JOB];
            np = h[H_NP];
            nt = h[H_NT];
            t = h[H_T];
            nrow = *reinterpret_cast<const int4 *>(
                st + (lane < 16 ? BatchStage::kn : BatchStage::vn) + cand * 256 +
                (lane & 15) * 16);
          }
          const float *SC = reinterpret_cast<const float *>(st + BatchStage::sc) +
                            cand * kBlockRows;
          if (!(flags & F_TAIL)) {
            // Prefix rows [first, first + rows), shared by every candidate.
            for (int r = lane; r < rows; r += 32) GSC[first + r] = SC[r];
            for (int t0 = 0; t0 < rows; t0 += kGroupTiles * kBox) {
              const uint32_t off = t0 * 128;
              tile_group(st + BatchStage::k0 + off, st + BatchStage::k1 + off,
                         st + BatchStage::v0 + off, st + BatchStage::v1 + off,
                         rows - t0, qb, p.scale_log2e, LG, first + t0, m0, m1,
                         l0, l1, o, lane);
            }
          } else {
            // This candidate's tail rows [first, first + rows) (+ the new row)
            // at block rows cand * T + ....
            const int live = rows + ((flags & F_NEW) ? 1 : 0);
            for (int r = lane; r < live; r += 32)
              GSC[np + first + r] = r < rows ? SC[r] : 0.f;
            if (flags & F_NEW) {
              const int rn = cand * T + (nt - first);
              const int ch = lane & 15, half = ch >> 3, cc = ch & 7;
              unsigned char *dst = st + (lane < 16 ? (half ? BatchStage::k1 : BatchStage::k0)
                                                   : (half ? BatchStage::v1 : BatchStage::v0));
              *reinterpret_cast<int4 *>(dst + rn * 128 + ((cc ^ (rn & 7)) << 4)) = nrow;
              wrote = true;
              __syncwarp();
            }
            for (int t0 = 0; t0 < live; t0 += kGroupTiles * kBox) {
              const uint32_t off = (cand * T + t0) * 128;
              tile_group(st + BatchStage::k0 + off, st + BatchStage::k1 + off,
                         st + BatchStage::v0 + off, st + BatchStage::v1 + off,
                         live - t0, qb, p.scale_log2e, LG, np + first + t0, m0,
                         m1, l0, l1, o, lane);
            }
          }
        }
        if (wrote) fence_proxy_async();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(smem_u32(&empty_bar[s]));
          if (cand == 0) consumed_n = seq + 1;
        }
        ++seq;
        if (flags & F_LAST) break;
      }
      if (stop || skip) continue;

      // ---- the candidate's back part: output, scores, append ----
#pragma unroll
      for (int off = 4; off < 32; off <<= 1) {
        l0 += __shfl_xor_sync(0xffffffffu, l0, off);
        l1 += __shfl_xor_sync(0xffffffffu, l1, off);
      }
      const float i0 = rcp(l0), i1 = rcp(l1);
      if (lane < 4 && !(l0 > 0.5f && l0 < INFINITY && l1 > 0.5f && l1 < INFINITY))
        atomicOr(c.err, ERR_NONFINITE);
      const Unit u = unit_of(p, idx);
      const size_t orow = (size_t)cand * per + u.row0;
      const size_t cu = (size_t)cand * units + u.ug;
      {
        constexpr int osz = kOutBf16 ? 2 : 4;
        unsigned char *gout = reinterpret_cast<unsigned char *>(p.out) + orow * G * 128 * osz;
#pragma unroll
        for (int mt = 0; mt < 8; ++mt) {
          if (kOutBf16) {
            const uint32_t lo = movm_t(pack_bf16(o[mt][0] * i0, o[mt][1] * i1));
            const uint32_t hi = movm_t(pack_bf16(o[mt][2] * i0, o[mt][3] * i1));
            const int g = lane >> 2, dd = 16 * mt + 2 * (lane & 3);
            if (g < G) {
              *reinterpret_cast<uint32_t *>(gout + ((size_t)g * 128 + dd) * 2) = lo;
              *reinterpret_cast<uint32_t *>(gout + ((size_t)g * 128 + dd + 8) * 2) = hi;
            }
          } else {
            float *of = reinterpret_cast<float *>(gout);
            const int d0 = 16 * mt + r0l;
            if (c2 < G) {
              of[c2 * 128 + d0] = o[mt][0] * i0;
              of[c2 * 128 + d0 + 8] = o[mt][2] * i0;
            }
            if (c2 + 1 < G) {
              of[(c2 + 1) * 128 + d0] = o[mt][1] * i1;
              of[(c2 + 1) * 128 + d0 + 8] = o[mt][3] * i1;
            }
          }
        }
      }
      // Per head: the maximum and 1 / sum (lanes 0..3 hold heads 2l, 2l+1).
      float Mg[8], iL[8];
#pragma unroll
      for (int g = 0; g < 8; ++g) {
        Mg[g] = __shfl_sync(0xffffffffu, (g & 1) ? m1 : m0, g >> 1);
        iL[g] = __shfl_sync(0xffffffffu, (g & 1) ? i1 : i0, g >> 1);
      }
      __syncwarp();  // this warp's logits and old scores are visible
      float *ps = f.pscore + cu * c.sstride;
      float *ts = f.tscore + cu * f.tstride;
      const int ntot = np + nt + 1;
      for (int r = lane; r < ntot; r += 32) {
        const float4 la = *reinterpret_cast<const float4 *>(LG + r * 8);
        const float4 lb = *reinterpret_cast<const float4 *>(LG + r * 8 + 4);
        const float lg8[8] = {la.x, la.y, la.z, la.w, lb.x, lb.y, lb.z, lb.w};
        float acc = 0.f;
#pragma unroll
        for (int g = 0; g < 8; ++g)
          if (g < G) acc += ex2(lg8[g] - Mg[g]) * iL[g];
        const float sc = GSC[r] + acc * p.inv_g;
        if (r < np) ps[r] = sc;
        else ts[r - np] = sc;
      }
      __nv_bfloat16 *dst = reinterpret_cast<__nv_bfloat16 *>(lane < 16 ? f.TK : f.TV) +
                           (cu * (size_t)f.tcap + nt) * 128;
      reinterpret_cast<int4 *>(dst)[lane & 15] = nrow;
      if (lane == 0) {
        f.tpos[cu * f.tstride + nt] = t;
        f.tlen[cu] = nt + 1;
      }
      __syncwarp();  // the area is reused by the next unit
    }
  }
  __syncthreads();
  // After an abort, wait (bounded) for copies still landing in the ring.
  if (s_abort && threadIdx.x == 0) {
    volatile int never = 0;
    for (int q = consumed_n; q < issued_n; ++q)
      mbar_wait(smem_u32(&full_bar[q % kStages]), (uint32_t)(q / kStages) & 1u,
                &never);
  }
}

}  // namespace

int fork_batch_max_cand() { return kMaxCand; }
int fork_batch_prefix_box_rows() { return kBlockRows; }
int fork_batch_tail_rows(int n_cand) {
  return n_cand >= 1 && n_cand <= kMaxCand ? tail_rows(n_cand) : 0;
}
size_t fork_batch_smem_bytes(int n_max, int n_cand) {
  return (size_t)kStages * BatchStage::bytes +
         (size_t)n_cand * warp_area_bytes(n_max) + 1024;
}

cudaError_t launch_fork_batch(const CUtensorMap &tmK, const CUtensorMap &tmV,
                              const CUtensorMap &tmK128,
                              const CUtensorMap &tmV128,
                              const CUtensorMap &tmTK, const CUtensorMap &tmTV,
                              const ForkBatchParams &p, int grid,
                              cudaStream_t st) {
  if (p.f.N < 1 || p.f.N > kMaxCand || p.f.p.G > 8 || p.n_max < 1)
    return cudaErrorInvalidValue;
  const size_t smem = fork_batch_smem_bytes(p.n_max, p.f.N);
  auto kern = p.f.p.out_bf16 ? fork_batch_kernel<true> : fork_batch_kernel<false>;
  cudaError_t e = cudaFuncSetAttribute(
      kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(kern, dim3(grid), dim3(32 * (p.f.N + 1)), smem, st, tmK,
                    tmV, tmK128, tmV128, tmTK, tmTV, p);
}

}  // namespace kvr
