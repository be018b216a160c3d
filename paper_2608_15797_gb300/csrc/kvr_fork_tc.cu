// kvr_fork_tc.cu -- the candidate-batched decode step of stepwise best-of-N
// (Sec. 2.2 Eq. 2, App. C) on 5th-generation tensor cores.  N candidates
// share the parent's live rows as a read-only prefix and each has a private
// tail.  Per candidate: append + Attn(q_t, C) (Eq. 1) over prefix + tail +
// new row, the candidate's accumulated attention (Sec. 2.1, mean over the G
// heads) of every row, and the new row appended to the tail (eviction is
// deferred to the commit).  bf16, head_dim 128, G <= 8, N <= 8, at most
// kMaxPrefix parent rows and kMaxTail tail rows before the append.
//
// Design (GB300, sm_103a).  A tcgen05.mma takes the tensor pipe about the
// same time for any N up to 64 (M = 128, K = 16), so the kernel is laid out
// to issue few, wide MMAs:
//  - The unit's N x G query rows are the M side (candidate c, head g at TMEM
//    lane (c & 1) * 32 + (c >> 1) * 8 + g of the unit's 64-lane slot).  S =
//    Q K^T over the shared prefix is one chain of 8 MMAs whatever N is.
//  - Tails are read per candidate pair, both tails contiguous in shared
//    memory: one MMA chain (N = twice the tail rows) computes the pair's
//    logits, with every lane outside the pair disabled (the MMA's
//    disable-output-lane mask), so all pairs share the same columns.  Even
//    candidates sit in lane quarter 0 of the slot and read the first half
//    of those columns, odd ones quarter 1 and the second half.
//  - PV per candidate tail (K = its rows, N = all 128 head-dim columns) with
//    the lanes of the other candidates disabled; P (bf16 hi and lo terms) is
//    the A operand, read straight from tensor memory.  The new rows (one per
//    candidate) are done on the CUDA cores: their logit is a 128-term dot
//    product and their PV term one multiply-add per output element.
//  - Two units are in flight, in the two 64-lane halves of tensor memory;
//    every MMA disables the other slot's lanes.  Per slot the columns hold S
//    (then P in its place, bf16 hi and lo terms) and O.
//  - Warp roles (12 warps, one CTA per SM): a K producer (by cp.async the
//    query rows into the slot's query buffer and the new rows and a header
//    into one of three buffers; K items by TMA), a V producer, an S issuer,
//    a PV issuer, and eight softmax/epilogue warps, two per TMEM lane
//    quarter, each taking alternate 16-column chunks of its rows.  K and V
//    stream through two rings of 8 KB slots (the V ring holds about a
//    unit's V, loaded while the unit's softmax runs); an item (the prefix,
//    or a candidate pair's tails, both head-dim halves) takes consecutive
//    slots.
//  - The softmax is exact: each warp reads its chunks of S from tensor
//    memory once, the two warps of a quarter exchange (max, sum), and the
//    probabilities go to P for PV and, in fp32, summed over a candidate's G
//    rows by a butterfly over its 8 lanes, to the score update.
//  - V rows past the live ones must be finite (their probabilities are zero,
//    but the memory may hold anything): the tail maps end at the live rows,
//    so TMA fills the rest with zeros, and a prefix box's extra rows are
//    zeroed in shared memory before PV reads them.  Every wait is bounded; on
//    timeout the kernel sets ERR_TIMEOUT, drains its copies and tensor work,
//    and returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <math.h>
#include <stdint.h>

#include "kvr_internal.h"
#include "kvr_ptx.cuh"

namespace kvr {
namespace {

using namespace ptx;

constexpr int kMaxCand = 8;
constexpr int kMaxPrefix = 128;  // parent rows per unit
constexpr int kMaxTail = 64;     // tail rows per candidate before the append
constexpr int kBox = 16;         // rows per prefix TMA box
constexpr int kSlot = 8192;      // ring slot bytes
constexpr int kSlotsK = 12, kSlotsV = 10;
constexpr int kHeads = 3;        // new-row buffers (unit k uses k % 3)
constexpr int kWarps = 12, kThreads = 32 * kWarps;
constexpr int kFirstCompute = 4;

// Tensor memory columns of a unit slot (within the slot's 64 lanes).  P
// replaces S in place: the 16 columns of a 16-key chunk take its 8 hi and
// then 8 lo columns of bf16 pairs (one thread reads and writes each chunk).
constexpr uint32_t kColSP = 0;    // S / P prefix [0,128)
constexpr uint32_t kColST = 128;  // S / P tail [128,256): a pair's two tails side by side
constexpr uint32_t kColO = 256;   // O [256,384)
constexpr uint32_t kTmemCols = 512;

// Per unit slot ts a query buffer (the unit's rows, [2][64][128 B], K-major,
// 128B swizzle), used by units ts, ts + 2, ...; per unit k % 3 a buffer of
// the new rows and a header.  The two query buffers are adjacent: each
// query descriptor reads 128 rows, of which slot 0's rows 64..127 lie in
// the 8 KB after its own rows and slot 1's rows 0..63 in the 8 KB before.
struct Nv {
  static constexpr int kn = 0;             // [8][256 B] new keys
  static constexpr int vn = 2048;          // [8][256 B] new values
  static constexpr int hdr = 4096;         // header words
  static constexpr int bytes = 5120;
};
enum : int { HD_IDX = 0, HD_NP, HD_NT, HD_POS, HD_OK };

struct Smem {  // offsets from the 1024-byte aligned base
  static constexpr int q = 0;                        // [2 slots][16 KB]
  static constexpr int nv = q + 2 * 16384;
  static constexpr int ringK = nv + kHeads * Nv::bytes;
  static constexpr int ringV = ringK + kSlotsK * kSlot;
  static constexpr int bytes = ringV + kSlotsV * kSlot;
  static constexpr int alloc = bytes + 1024;
};
static_assert(Smem::ringK % 1024 == 0, "ring slots stay 1024-byte aligned");
static_assert(kSlotsK <= 32 && kSlotsV <= 32, "slot phases are bit masks");
static_assert(2 * kMaxTail * 256 <= 4 * kSlot && kMaxPrefix * 256 <= 4 * kSlot &&
                  4 <= kSlotsK && 4 <= kSlotsV,
              "an item takes at most 4 slots, and fits in either ring");

// The tensor maps: the parent's K and V slabs in 16-row boxes, and the
// call's tails as {128, nt, units, N} (nt: the rows every tail holds before
// the append, so rows past them read as zeros) with boxes {64, t16, 1,
// min(N, 2)}, t16 = nt rounded up to 16.
struct TcMaps {
  CUtensorMap k, v, tk, tv;
};

// ---- tensor-core helpers specific to this kernel -------------------------
// D[tmem] (+)= A[smem] * B[smem] on the lanes not set in the mask words
// (bit i of word w disables lane 32 w + i).
__device__ __forceinline__ void mma_ss(uint32_t d, uint64_t a, uint64_t b,
                                       uint32_t id, uint32_t m0, uint32_t m1,
                                       uint32_t m2, uint32_t m3, uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %8, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, {%4, %5, %6, %7}, p;\n\t}" ::"r"(d),
      "l"(a), "l"(b), "r"(id), "r"(m0), "r"(m1), "r"(m2), "r"(m3), "r"(acc)
      : "memory");
}
// The same with A read from tensor memory (bf16 pairs, the lower k in the
// low half of each 32-bit column).
__device__ __forceinline__ void mma_ts(uint32_t d, uint32_t a, uint64_t b,
                                       uint32_t id, uint32_t m0, uint32_t m1,
                                       uint32_t m2, uint32_t m3, uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %8, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, {%4, %5, %6, %7}, p;\n\t}" ::"r"(d),
      "r"(a), "l"(b), "r"(id), "r"(m0), "r"(m1), "r"(m2), "r"(m3), "r"(acc)
      : "memory");
}
__device__ __forceinline__ void tmem_st8(uint32_t taddr, const uint32_t (&v)[8]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"r"(taddr),
      "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]),
      "r"(v[7])
      : "memory");
}
__device__ __forceinline__ void tmem_wait_st() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void named_bar(int id, int threads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}
// Named barrier that also ANDs a predicate over the participating threads.
__device__ __forceinline__ bool named_bar_and(int id, int threads, bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred pi, po;\n\tsetp.ne.b32 pi, %1, 0;\n\t"
      "bar.red.and.pred po, %2, %3, pi;\n\tselp.u32 %0, 1, 0, po;\n\t}"
      : "=r"(r)
      : "r"(v ? 1 : 0), "r"(id), "r"(threads)
      : "memory");
  return r != 0;
}

// TMEM lane (within the slot) of candidate c's first row, and the disabled-
// lane words of one slot, one candidate or one candidate pair.
__device__ __forceinline__ int cand_row(int c) { return (c & 1) * 32 + (c >> 1) * 8; }
struct Mask {
  uint32_t w[4];
};
__device__ __forceinline__ Mask slot_mask(int ts) {
  Mask m;
  m.w[0] = m.w[1] = ts ? 0xFFFFFFFFu : 0u;
  m.w[2] = m.w[3] = ts ? 0u : 0xFFFFFFFFu;
  return m;
}
__device__ __forceinline__ Mask cand_mask(int ts, int c) {
  Mask m;
  m.w[0] = m.w[1] = m.w[2] = m.w[3] = 0xFFFFFFFFu;
  m.w[2 * ts + (c & 1)] = ~(0xFFu << (8 * (c >> 1)));
  return m;
}
__device__ __forceinline__ Mask pair_mask(int ts, int pm) {
  Mask m;
  m.w[0] = m.w[1] = m.w[2] = m.w[3] = 0xFFFFFFFFu;
  m.w[2 * ts] = m.w[2 * ts + 1] = ~(0xFFu << (8 * pm));
  return m;
}

struct Unit {
  size_t ug;    // the parent's unit
  size_t row0;  // unit row of the call ([S][nl][H])
};
__device__ __forceinline__ Unit unit_of(const ForkTcParams &p, int idx) {
  const CacheView &c = p.f.p;
  const int h = idx % c.H, lr = (idx / c.H) % p.nl, sq = idx / (c.H * p.nl);
  Unit u;
  u.ug = ((size_t)sq * c.L + p.lb + lr) * c.H + h;
  u.row0 = ((size_t)sq * p.nl + lr) * c.H + h;
  return u;
}

// Shared state of one CTA.
struct Ctl {
  uint64_t fullK[kSlotsK], emptyK[kSlotsK], fullV[kSlotsV], emptyV[kSlotsV];
  // head_full[k % 3]: unit k's query rows (query buffer k & 1), new rows and
  // header have landed; head_free[k % 3]: its new rows are no longer read;
  // q_free[ts]: slot ts's query rows are no longer read (S done and the
  // new rows' logits taken).
  uint64_t head_full[kHeads], head_free[kHeads], q_free[2];
  uint64_t s_full[2], p_full[2], o_full[2], o_free[2], drain[2];
  float2 xch[4][2][32];   // (max, sum) of the two warps of each quarter
  // Items issued (by the producers) and waited for (by the issuers), and
  // each item's first slot and full-barrier parity, for the drain after an
  // abort (at most one item per slot is outstanding).
  int issuedK, consumedK, issuedV, consumedV;
  int logK[kSlotsK], logV[kSlotsV];
  uint32_t tmem;
  int abort;
};

// Bounded wait that raises the CTA's abort flag (and ERR_TIMEOUT) when it
// runs out; false when it or another warp gave up.  Each lane waits on its
// own; warp_wait makes the answer the same for the whole warp.
__device__ __forceinline__ bool wait_or_abort(uint64_t *bar, uint32_t parity,
                                              Ctl &s, unsigned *err,
                                              uint64_t limit) {
  volatile int *ab = &s.abort;
  if (mbar_wait(smem_u32(bar), parity, ab, limit)) return true;
  if (!*ab) {
    atomicOr(err, ERR_TIMEOUT);
    *ab = 1;
  }
  return false;
}
__device__ __forceinline__ bool warp_wait(uint64_t *bar, uint32_t parity, Ctl &s,
                                          unsigned *err, uint64_t limit) {
  return __all_sync(0xffffffffu, wait_or_abort(bar, parity, s, err, limit)) != 0;
}

// A ring of kSlots 8 KB slots; an item takes n consecutive slots (wrapping
// to slot 0 when it would pass the end), and the barriers of its first slot
// stand for it: all of its copies arrive on that full barrier, and its
// issuer releases it with one commit on that empty barrier.  Producer and
// consumer walk the same items in the same order, so each side tracks by
// itself the slots and the parities of the barriers it waits on.
template <int kSlots>
struct RingPos {
  int next = 0;
  uint32_t full_ph = 0;  // parity bit of every slot's next full wait
  __device__ __forceinline__ int take(int n) {
    if (next + n > kSlots) next = 0;
    const int s = next;
    next += n;
    return s;
  }
};
// The producer's view (lane 0): which item holds each slot, to wait for
// the release of every item a new one overlaps.
template <int kSlots>
struct RingOwn {
  signed char first[kSlots];  // first slot of the holding item, -1 when free
  signed char len[kSlots];    // slots of the item starting here
  uint32_t rel_ph = 0;        // parity bit of every first slot's next release
  __device__ __forceinline__ void init() {
    for (int i = 0; i < kSlots; ++i) first[i] = -1;
  }
};
__device__ __forceinline__ int slots_for(int bytes) { return (bytes + kSlot - 1) / kSlot; }

// The unit's items: the prefix (both head-dim halves, np16 rows each) if
// np > 0, then one item per candidate pair holding both tails (t16 rows
// each, both halves) if nt > 0.
__device__ __forceinline__ int prefix_bytes(int np16) { return np16 * 256; }
__device__ __forceinline__ int pair_bytes(int t16) { return 2 * t16 * 256; }

// ---- producers (warps 0 and 3) ----------------------------------------------
// Claim the slots of the next item (`bytes` of layout; waiting until their
// previous uses are released) and post the `tx` bytes its copies deliver on
// the first slot's full barrier.
template <int kSlots>
__device__ bool put_item(RingPos<kSlots> &rp, RingOwn<kSlots> &own, uint64_t *full,
                         uint64_t *empty, int *log, int *issued, int bytes, int tx, Ctl &s,
                         unsigned *err, int lane, int &slot) {
  const int n = slots_for(bytes);
  slot = rp.take(n);
  int got = 1;
  if (lane == 0) {
    for (int i = 0; i < n && got; ++i) {
      const int f = own.first[slot + i];
      if (f < 0) continue;
      got = wait_or_abort(&empty[f], (own.rel_ph >> f) & 1u, s, err, kWaitNs);
      own.rel_ph ^= 1u << f;
      for (int j = 0; j < own.len[f]; ++j) own.first[f + j] = -1;
    }
    for (int i = 0; i < n; ++i) own.first[slot + i] = (signed char)slot;
    own.len[slot] = (signed char)n;
  }
  got = __shfl_sync(0xffffffffu, got, 0);
  if (!got) return false;
  const uint32_t fph = (rp.full_ph >> slot) & 1u;
  rp.full_ph ^= 1u << slot;
  if (lane == 0) {
    log[*issued % kSlots] = slot | (int)(fph << 8);
    *issued += 1;
    mbar_expect_tx(smem_u32(&full[slot]), (uint32_t)tx);
  }
  return true;
}

// Item `it` of a unit's K (or V): the prefix if it == -1, else the tails of
// candidate pair it.
template <int kSlots>
__device__ bool put_unit_item(RingPos<kSlots> &rp, RingOwn<kSlots> &own, uint64_t *full,
                              uint64_t *empty, int *log, int *issued, unsigned char *ring,
                              const CUtensorMap *slab, const CUtensorMap *tails,
                              const ForkTcParams &p, size_t ug, int np, int nt, int it,
                              Ctl &s, int lane) {
  const ForkView &f = p.f;
  const CacheView &c = f.p;
  const int np16 = (np + 15) & ~15, t16 = (nt + 15) & ~15;
  if (it < 0) {
    int slot;
    if (!put_item(rp, own, full, empty, log, issued, prefix_bytes(np16), prefix_bytes(np16),
                  s, c.err, lane, slot))
      return false;
    if (lane == 0) {
      const uint32_t dst = smem_u32(ring + slot * kSlot), bar = smem_u32(&full[slot]);
      for (int h = 0; h < 2; ++h)
        for (int b = 0; b < np16 / kBox; ++b)
          tma_load_2d(dst + h * np16 * 128 + b * kBox * 128, slab, 64 * h,
                      (int)(ug * (size_t)c.cap + (size_t)b * kBox), bar);
    }
    return true;
  }
  // A tail box holds min(N, 2) candidates (rows past N read as zeros).
  const int tx = 2 * min(f.N, 2) * t16 * 128;
  int slot;
  if (!put_item(rp, own, full, empty, log, issued, pair_bytes(t16), tx, s, c.err, lane, slot))
    return false;
  if (lane == 0) {
    const uint32_t dst = smem_u32(ring + slot * kSlot), bar = smem_u32(&full[slot]);
    for (int h = 0; h < 2; ++h)
      tma_load_4d(dst + h * 2 * t16 * 128, tails, 64 * h, 0, (int)ug, 2 * it, bar);
  }
  return true;
}
// Item numbers of a unit: -1 (the prefix) when np > 0, then 0 .. pairs - 1.
__device__ __forceinline__ int first_item(int np) { return np > 0 ? -1 : 0; }
__device__ __forceinline__ int end_item(int nt, int N) { return nt > 0 ? (N + 1) / 2 : 0; }

// The unit's K (or V) items.
template <int kSlots>
__device__ bool unit_items(RingPos<kSlots> &rp, RingOwn<kSlots> &own, uint64_t *full,
                           uint64_t *empty, int *log, int *issued, unsigned char *ring,
                           const CUtensorMap *slab, const CUtensorMap *tails,
                           const ForkTcParams &p, size_t ug, int np, int nt, Ctl &s,
                           int lane) {
  for (int it = first_item(np); it < end_item(nt, p.f.N); ++it)
    if (!put_unit_item(rp, own, full, empty, log, issued, ring, slab, tails, p, ug, np, nt, it,
                       s, lane))
      return false;
  return true;
}

// Non-blocking test of an mbarrier phase.
__device__ __forceinline__ bool mbar_test(uint64_t *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// What the K producer keeps of a unit whose head it has loaded.
struct HeadInfo {
  size_t ug;
  int np, nt, ok;
};

__device__ void produce_k(const ForkTcParams &p, const TcMaps &m,
                          unsigned char *smem, Ctl &s, int mine, int lane) {
  const ForkView &f = p.f;
  const CacheView &c = f.p;
  const int N = f.N, G = c.G;
  const size_t units = (size_t)c.S * c.L * c.H;
  const size_t per = (size_t)c.S * p.nl * c.H;  // unit rows of the call
  RingPos<kSlotsK> rp;
  RingOwn<kSlotsK> own;
  own.init();
  // The head of unit k: query rows into slot k & 1's query buffer, new rows
  // and header into buffer k % 3, once both are free.  With block false it
  // only goes ahead when they are free already.  1: loaded, 0: not yet,
  // -1: a wait gave up.
  auto load_head = [&](int k, bool block, HeadInfo &hi) -> int {
    const int hb = k % kHeads, ts = k & 1;
    const uint32_t ph_h = ((uint32_t)(k / kHeads) & 1u) ^ 1u;
    const uint32_t ph_q = ((uint32_t)(k >> 1) & 1u) ^ 1u;
    int got = 1;
    if (lane == 0) {
      if (block)
        got = wait_or_abort(&s.head_free[hb], ph_h, s, c.err, kWaitNs) &&
              wait_or_abort(&s.q_free[ts], ph_q, s, c.err, kWaitNs) ? 1 : -1;
      else
        got = mbar_test(&s.head_free[hb], ph_h) && mbar_test(&s.q_free[ts], ph_q) ? 1 : 0;
    }
    got = __shfl_sync(0xffffffffu, got, 0);
    if (got != 1) return got;
    const int idx = (int)blockIdx.x + k * (int)gridDim.x;
    const Unit u = unit_of(p, idx);
    const int np = c.state[4 * u.ug], bp = c.state[4 * u.ug + 1];
    // Every candidate's tail has the same length (one row per call each).
    const int mynt = lane < N ? f.tlen[(size_t)lane * units + u.ug] : -1;
    const int nt = __shfl_sync(0xffffffffu, mynt, 0);
    const bool same = __all_sync(0xffffffffu, lane >= N || mynt == nt);
    const bool ok = same && np >= 0 && np <= kMaxPrefix && np <= c.cap &&
                    nt == p.nt && nt <= kMaxTail && nt + 1 <= f.tcap;
    if (!ok && lane == 0)
      atomicOr(c.err, (same && nt + 1 > f.tcap) ? ERR_CAPACITY : ERR_LENGTH);
    unsigned char *hd = smem + Smem::nv + hb * Nv::bytes;
    const uint32_t h0 = smem_u32(hd), q0 = smem_u32(smem + Smem::q + ts * 16384);
    if (ok) {
      // Query rows at their TMEM lanes (16-byte pieces, 128B swizzle).
      for (int i = lane; i < N * G * 16; i += 32) {
        const int row = i >> 4, ch = i & 15;
        const int cand = row / G, g = row % G, r = cand_row(cand) + g;
        const __nv_bfloat16 *src =
            p.q + (((size_t)cand * per + u.row0) * G + g) * 128 + ch * 8;
        cp_async16(q0 + (ch >> 3) * 8192 + r * 128 + (((ch & 7) ^ (r & 7)) << 4), src);
      }
      // New key and value rows of every candidate (plain rows).
      for (int i = lane; i < N * 32; i += 32) {
        const int cand = i >> 5, ch = i & 15;
        const bool v = (i & 16) != 0;
        const __nv_bfloat16 *src =
            (v ? p.v_new : p.k_new) + ((size_t)cand * per + u.row0) * 128 + ch * 8;
        cp_async16(h0 + (v ? Nv::vn : Nv::kn) + cand * 256 + ch * 16, src);
      }
    }
    if (lane == 0) {
      int *hw = reinterpret_cast<int *>(hd + Nv::hdr);
      hw[HD_IDX] = idx;
      hw[HD_NP] = np;
      hw[HD_NT] = nt;
      hw[HD_POS] = bp + nt;
      hw[HD_OK] = ok ? 1 : 0;
      mbar_arrive(smem_u32(&s.head_full[hb]));
    }
    cp_async_arrive_noinc(smem_u32(&s.head_full[hb]));
    hi.ug = u.ug;
    hi.np = np;
    hi.nt = nt;
    hi.ok = ok;
    return 1;
  };
  // Heads run one unit ahead of the K items when their buffers allow it,
  // so that a unit's S can start as soon as its first K item lands.
  HeadInfo cur{}, nxt{};
  int loaded = 0;  // heads loaded so far
  if (mine > 0) {
    if (load_head(0, true, cur) != 1) mine = 0;
    loaded = 1;
  }
  bool fine = true;
  for (int k = 0; k < mine && fine; ++k) {
    for (int it = cur.ok ? first_item(cur.np) : 0; cur.ok && it < end_item(cur.nt, N); ++it) {
      if (loaded == k + 1 && k + 1 < mine) {  // the next head, if its buffers are free
        const int r = load_head(k + 1, false, nxt);
        if (r < 0) {
          fine = false;
          break;
        }
        loaded += r;
      }
      if (!(fine = put_unit_item(rp, own, s.fullK, s.emptyK, s.logK, &s.issuedK,
                                 smem + Smem::ringK, &m.k, &m.tk, p, cur.ug, cur.np, cur.nt,
                                 it, s, lane)))
        break;
    }
    if (!fine) break;
    if (k + 1 < mine) {
      if (loaded == k + 1) {
        if (load_head(k + 1, true, nxt) != 1) break;
        loaded += 1;
      }
      cur = nxt;
    }
  }
  asm volatile("cp.async.wait_all;" ::: "memory");
}

__device__ void produce_v(const ForkTcParams &p, const TcMaps &m,
                          unsigned char *smem, Ctl &s, int mine, int lane) {
  const CacheView &c = p.f.p;
  RingPos<kSlotsV> rp;
  RingOwn<kSlotsV> own;
  own.init();
  for (int k = 0; k < mine; ++k) {
    const int hb = k % kHeads;
    if (!warp_wait(&s.head_full[hb], (uint32_t)(k / kHeads) & 1u, s, c.err, kWaitNs)) break;
    // V of unit k is needed once its softmax is done: start the copies when
    // its S is done, so they land while the softmax runs.
    if (!warp_wait(&s.s_full[k & 1], (uint32_t)(k >> 1) & 1u, s, c.err, kWaitNs)) break;
    const int *hw = reinterpret_cast<const int *>(smem + Smem::nv + hb * Nv::bytes + Nv::hdr);
    const int idx = hw[HD_IDX], np = hw[HD_NP], nt = hw[HD_NT], ok = hw[HD_OK];
    if (ok && !unit_items(rp, own, s.fullV, s.emptyV, s.logV, &s.issuedV, smem + Smem::ringV,
                          &m.v, &m.tv, p, unit_of(p, idx).ug, np, nt, s, lane))
      break;
  }
}

// ---- MMA issuers (warps 1 and 2) ------------------------------------------------
// Wait for the next item of a ring (every lane: the V items are patched in
// shared memory by the whole warp); release it once its MMAs are done.
template <int kSlots>
__device__ __forceinline__ bool get_item(RingPos<kSlots> &rp, uint64_t *full, int *consumed,
                                         int bytes, Ctl &s, unsigned *err, uint64_t lim,
                                         int lane, int &slot) {
  slot = rp.take(slots_for(bytes));
  const bool ok = warp_wait(&full[slot], (rp.full_ph >> slot) & 1u, s, err, lim);
  rp.full_ph ^= 1u << slot;
  if (ok && lane == 0) *consumed += 1;
  return ok;
}
__device__ __forceinline__ void release_item(uint64_t *empty, int slot, int lane) {
  if (lane == 0) tc_commit(smem_u32(&empty[slot]));
}

__device__ void issue_s(const ForkTcParams &p, unsigned char *smem, Ctl &s, int mine,
                        int lane) {
  const CacheView &c = p.f.p;
  const int N = p.f.N;
  const uint32_t tm = s.tmem;
  const uint64_t lim = c.wait_ns;
  RingPos<kSlotsK> rp;
  unsigned char *ring = smem + Smem::ringK;
  for (int k = 0; k < mine; ++k) {
    const int hb = k % kHeads, ts = k & 1;
    if (!warp_wait(&s.head_full[hb], (uint32_t)(k / kHeads) & 1u, s, c.err, kWaitNs)) break;
    // PV of unit k - 2 (same slot) is done: its P, in S's columns, is read.
    if (!warp_wait(&s.o_full[ts], ((uint32_t)(k >> 1) & 1u) ^ 1u, s, c.err, kWaitNs)) break;
    const int *hw = reinterpret_cast<const int *>(smem + Smem::nv + hb * Nv::bytes + Nv::hdr);
    const int np = hw[HD_NP], nt = hw[HD_NT], ok = hw[HD_OK];
    fence_proxy_async();  // the query rows came by cp.async (generic proxy)
    tc_fence_after();
    // Query descriptor: slot 1's rows are A rows 64..127, so its base sits
    // 8 KB (64 rows) before its buffer's first row.  Offsets below are in
    // the descriptor's 16-byte units: 16 head-dim columns = 2, a 64-column
    // half = 512 in Q (8 KB) and rows * 8 in K.
    const uint64_t qd = sdesc_sw128(smem_u32(smem + Smem::q + ts * 16384) - (uint32_t)ts * 8192u,
                                    16, 1024);
    bool fine = true;
    if (ok) {
      const int np16 = (np + 15) & ~15, t16 = (nt + 15) & ~15;
      if (np16 > 0) {
        int slot;
        if (!(fine = get_item(rp, s.fullK, &s.consumedK, prefix_bytes(np16), s, c.err, lim,
                              lane, slot)))
          break;
        tc_fence_after();
        if (lane == 0) {
          const Mask ms = slot_mask(ts);
          const uint32_t id = idesc_bf16(128, np16, false);
          const uint64_t kd = sdesc_sw128(smem_u32(ring + slot * kSlot), 16, 1024);
#pragma unroll
          for (int kk = 0; kk < 8; ++kk)
            mma_ss(tm + kColSP, qd + (uint64_t)((kk >> 2) * 512 + (kk & 3) * 2),
                   kd + (uint64_t)((kk >> 2) * np16 * 8 + (kk & 3) * 2), id, ms.w[0], ms.w[1],
                   ms.w[2], ms.w[3], kk > 0);
        }
        __syncwarp();
        release_item(s.emptyK, slot, lane);
      }
      for (int pm = 0; t16 > 0 && pm < (N + 1) / 2; ++pm) {
        int slot;
        if (!(fine = get_item(rp, s.fullK, &s.consumedK, pair_bytes(t16), s, c.err, lim, lane,
                              slot)))
          break;
        tc_fence_after();
        if (lane == 0) {
          const Mask mp = pair_mask(ts, pm);
          const uint32_t id = idesc_bf16(128, 2 * t16, false);
          const uint64_t kd = sdesc_sw128(smem_u32(ring + slot * kSlot), 16, 1024);
#pragma unroll
          for (int kk = 0; kk < 8; ++kk)
            mma_ss(tm + kColST, qd + (uint64_t)((kk >> 2) * 512 + (kk & 3) * 2),
                   kd + (uint64_t)((kk >> 2) * 2 * t16 * 8 + (kk & 3) * 2), id, mp.w[0],
                   mp.w[1], mp.w[2], mp.w[3], kk > 0);
        }
        __syncwarp();
        release_item(s.emptyK, slot, lane);
      }
      if (!fine) break;
    }
    if (lane == 0) {
      tc_commit(smem_u32(&s.s_full[ts]));
      tc_commit(smem_u32(&s.q_free[ts]));
    }
    __syncwarp();
  }
  // Tensor work still in flight completes before the CTA frees its memory.
  if (lane == 0) {
    tc_commit(smem_u32(&s.drain[0]));
    volatile int never = 0;
    mbar_wait(smem_u32(&s.drain[0]), 0, &never);
  }
  __syncwarp();
}

__device__ void issue_pv(const ForkTcParams &p, unsigned char *smem, Ctl &s, int mine,
                         int lane) {
  const CacheView &c = p.f.p;
  const int N = p.f.N;
  const uint32_t tm = s.tmem;
  const uint64_t lim = c.wait_ns;
  RingPos<kSlotsV> rp;
  unsigned char *ring = smem + Smem::ringV;
  const uint32_t id_pv = idesc_bf16(128, 128, true);
  for (int k = 0; k < mine; ++k) {
    const int hb = k % kHeads, ts = k & 1;
    if (!warp_wait(&s.head_full[hb], (uint32_t)(k / kHeads) & 1u, s, c.err, kWaitNs)) break;
    if (!warp_wait(&s.p_full[ts], (uint32_t)(k >> 1) & 1u, s, c.err, kWaitNs)) break;
    // O of unit k - 2 (same slot) has been read.
    if (!warp_wait(&s.o_free[ts], ((uint32_t)(k >> 1) & 1u) ^ 1u, s, c.err, kWaitNs)) break;
    tc_fence_after();
    const int *hw = reinterpret_cast<const int *>(smem + Smem::nv + hb * Nv::bytes + Nv::hdr);
    const int np = hw[HD_NP], nt = hw[HD_NT], ok = hw[HD_OK];
    bool fine = true;
    if (ok) {
      const int np16 = (np + 15) & ~15, t16 = (nt + 15) & ~15;
      if (np16 > 0) {
        int slot;
        if (!(fine = get_item(rp, s.fullV, &s.consumedV, prefix_bytes(np16), s, c.err, lim,
                              lane, slot)))
          break;
        unsigned char *it = ring + slot * kSlot;
        if (np < np16) {  // rows [np, np16) of both halves are not live
          for (int i = np * 8 + lane; i < np16 * 8; i += 32) {
            *reinterpret_cast<int4 *>(it + i * 16) = make_int4(0, 0, 0, 0);
            *reinterpret_cast<int4 *>(it + np16 * 128 + i * 16) = make_int4(0, 0, 0, 0);
          }
          fence_proxy_async();
        }
        __syncwarp();
        tc_fence_after();
        if (lane == 0) {
          const Mask ms = slot_mask(ts);
          // MN-major V: the two 64-column halves np16 * 128 bytes apart; 16
          // rows (one K step) = 2048 bytes = 128 descriptor units.
          const uint64_t vd = sdesc_sw128(smem_u32(it), np16 * 128, 1024);
          for (int kk = 0; kk < np16 / 16; ++kk) {
            const uint64_t b = vd + (uint64_t)(kk * 128);
            mma_ts(tm + kColO, tm + kColSP + 16 * kk, b, id_pv, ms.w[0], ms.w[1], ms.w[2],
                   ms.w[3], kk > 0);
            mma_ts(tm + kColO, tm + kColSP + 16 * kk + 8, b, id_pv, ms.w[0], ms.w[1],
                   ms.w[2], ms.w[3], 1);
          }
        }
        __syncwarp();
        release_item(s.emptyV, slot, lane);
      }
      for (int pm = 0; t16 > 0 && pm < (N + 1) / 2; ++pm) {
        int slot;
        if (!(fine = get_item(rp, s.fullV, &s.consumedV, pair_bytes(t16), s, c.err, lim, lane,
                              slot)))
          break;
        unsigned char *it = ring + slot * kSlot;  // tail rows past nt arrive as zeros
        tc_fence_after();
        if (lane == 0) {
          for (int cc = 0; cc < 2 && 2 * pm + cc < N; ++cc) {
            const Mask mc = cand_mask(ts, 2 * pm + cc);
            // Candidate cc's tail: t16 rows at cc * t16 * 128 in each half;
            // the halves 2 * t16 * 128 bytes apart.
            const uint64_t vd =
                sdesc_sw128(smem_u32(it) + cc * t16 * 128, 2 * t16 * 128, 1024);
            // Its P: the chunks of its parity's half of the pair's columns.
            const uint32_t pa = tm + kColST + (uint32_t)(cc * t16);
            for (int kk = 0; kk < t16 / 16; ++kk) {
              const uint64_t b = vd + (uint64_t)(kk * 128);
              mma_ts(tm + kColO, pa + 16 * kk, b, id_pv, mc.w[0], mc.w[1], mc.w[2], mc.w[3],
                     np16 > 0 || kk > 0);
              mma_ts(tm + kColO, pa + 16 * kk + 8, b, id_pv, mc.w[0], mc.w[1], mc.w[2],
                     mc.w[3], 1);
            }
          }
        }
        __syncwarp();
        release_item(s.emptyV, slot, lane);
      }
      if (!fine) break;
    }
    if (lane == 0) tc_commit(smem_u32(&s.o_full[ts]));
    __syncwarp();
  }
  if (lane == 0) {
    tc_commit(smem_u32(&s.drain[1]));
    volatile int never = 0;
    mbar_wait(smem_u32(&s.drain[1]), 0, &never);
  }
  __syncwarp();
}

// ---- softmax and epilogue (warps 4..11) ---------------------------------------
// Butterfly over the 8 lanes of a candidate: in: v[16] per lane (its row's
// values of 16 columns); out: the sums over the 8 rows of columns 2 r8 and
// 2 r8 + 1, r8 = lane % 8.
__device__ __forceinline__ float2 colsum8(const float (&v)[16], int r8) {
  const bool b2 = (r8 & 4) != 0, b1 = (r8 & 2) != 0, b0 = (r8 & 1) != 0;
  float a[8], b[4];
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const float send = b2 ? v[i] : v[i + 8];
    const float keep = b2 ? v[i + 8] : v[i];
    a[i] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float send = b1 ? a[i] : a[i + 4];
    const float keep = b1 ? a[i + 4] : a[i];
    b[i] = keep + __shfl_xor_sync(0xffffffffu, send, 2);
  }
  float r[2];
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const float send = b0 ? b[i] : b[i + 2];
    const float keep = b0 ? b[i + 2] : b[i];
    r[i] = keep + __shfl_xor_sync(0xffffffffu, send, 1);
  }
  return make_float2(r[0], r[1]);
}

// fp32 dot product of query row r (the head's 128B-swizzled rows) and a
// plain bf16 row of 128 elements.
__device__ __forceinline__ float dot_row(const unsigned char *q, int r,
                                         const unsigned char *kv) {
  float acc = 0.f;
#pragma unroll
  for (int ch = 0; ch < 16; ++ch) {
    const uint4 a = *reinterpret_cast<const uint4 *>(q + (ch >> 3) * 8192 + r * 128 +
                                                      (((ch & 7) ^ (r & 7)) << 4));
    const uint4 b = *reinterpret_cast<const uint4 *>(kv + ch * 16);
    const uint32_t av[4] = {a.x, a.y, a.z, a.w}, bv[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 x = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&av[j]));
      const float2 y = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&bv[j]));
      acc = fmaf(x.x, y.x, acc);
      acc = fmaf(x.y, y.y, acc);
    }
  }
  return acc;
}

// kOwn: 16-column chunks of S a warp holds at most (prefix and tail chunks
// alternate between the two warps of a quarter): 6 for the largest units
// (8 + 4 chunks), 5 when a call's units have at most 10.
template <bool kOutBf16, int kOwn>
__device__ void softmax_epilogue(const ForkTcParams &p, unsigned char *smem,
                                 Ctl &s, int mine, int warp, int lane) {
  const ForkView &f = p.f;
  const CacheView &c = f.p;
  const int N = f.N, G = c.G;
  const size_t units = (size_t)c.S * c.L * c.H;
  const size_t per = (size_t)c.S * p.nl * c.H;
  const int qq = warp & 3;                        // TMEM lane quarter
  const int ts = qq >> 1;                         // unit slot
  const int par = qq & 1;                         // candidates of this parity
  const int hh = (warp - kFirstCompute) >> 2;     // column half (alternate chunks)
  const int cand = ((lane >> 3) << 1) | par, g = lane & 7, r8 = lane & 7;
  const int r = par * 32 + lane;                  // row within the slot
  const bool cand_ok = cand < N;
  const bool real = cand_ok && g < G;
  const uint32_t trow = s.tmem + ((uint32_t)(qq * 32) << 16);
  const float scale = p.scale_log2e, inv_g = p.inv_g;
  const int bar_id = 1 + qq;                      // the two warps of this quarter
  // The two warps of a quarter meet at named barriers, so they leave the
  // loop together: a failed wait is carried to the next agreement point.
  bool alive = true;
  for (int k = ts; k < mine; k += 2) {
    const int hb = k % kHeads;
    const uint32_t ph = (uint32_t)(k >> 1) & 1u;
    alive = alive &&
            wait_or_abort(&s.head_full[hb], (uint32_t)(k / kHeads) & 1u, s, c.err, kWaitNs);
    const unsigned char *hd = smem + Smem::nv + hb * Nv::bytes;
    const unsigned char *qb = smem + Smem::q + ts * 16384;
    const int *hw = reinterpret_cast<const int *>(hd + Nv::hdr);
    const int idx = hw[HD_IDX], np = hw[HD_NP], nt = hw[HD_NT], pos = hw[HD_POS];
    const bool ok = alive && hw[HD_OK] != 0;
    const int nPB = (np + 15) >> 4, nT = (nt + 15) >> 4;
    const int nch = nPB + nT;
    const uint32_t col_t = kColST + (uint32_t)(par * 16 * nT);  // this parity's tail logits
    const Unit u = unit_of(p, idx);
    const size_t cu = (size_t)cand * units + u.ug;
    float *ps = f.pscore + cu * c.sstride;
    float *tsc = f.tscore + cu * f.tstride;
    // The new row's logit (CUDA cores), while the tensor work runs.
    float xn = -INFINITY;
    if (ok && real) xn = dot_row(qb, r, hd + Nv::kn + cand * 256) * scale;
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_u32(&s.q_free[ts]));  // this warp's query reads are done
    alive = alive && wait_or_abort(&s.s_full[ts], ph, s, c.err, kWaitNs);
    if (!named_bar_and(bar_id, 64, alive)) break;
    tc_fence_after();
    float pn = 0.f;
    if (ok) {
      // This warp's chunks of the scaled logits (base 2), all loads in
      // flight at once; masked past the live keys.
      float e[kOwn][16];
#pragma unroll
      for (int t = 0; t < kOwn; ++t) {
        const int i = 2 * t + hh;
        if (i < nch)
          tmem_ld16f_nowait(trow + (i < nPB ? kColSP + 16 * i : col_t + 16 * (i - nPB)), e[t]);
      }
      tmem_wait_ld();
      float mx = hh == 0 && real ? xn : -INFINITY;  // the first warp counts the new row
#pragma unroll
      for (int t = 0; t < kOwn; ++t) {
        const int i = 2 * t + hh;
        if (i < nch) {
          const int lim = i < nPB ? np - 16 * i : nt - 16 * (i - nPB);
#pragma unroll
          for (int jj = 0; jj < 16; ++jj) {
            e[t][jj] = jj < lim ? e[t][jj] * scale : -INFINITY;
            mx = fmaxf(mx, e[t][jj]);
          }
        }
      }
      const float ref = mx == -INFINITY ? 0.f : mx;
      float sm = hh == 0 && real ? ex2(xn - ref) : 0.f;
#pragma unroll
      for (int t = 0; t < kOwn; ++t) {
        const int i = 2 * t + hh;
        if (i < nch) {
#pragma unroll
          for (int jj = 0; jj < 16; ++jj) {
            e[t][jj] = ex2(e[t][jj] - ref);  // exp2(-inf) = 0 for masked keys
            sm += e[t][jj];
          }
        }
      }
      // Exchange (max, sum) with the other warp of this quarter.
      s.xch[qq][hh][lane] = make_float2(mx, sm);
      named_bar(bar_id, 64);
      const float2 o2 = s.xch[qq][hh ^ 1][lane];
      const float M = fmaxf(mx, o2.x);
      const float L = (mx == -INFINITY ? 0.f : sm * ex2(mx - M)) +
                      (o2.x == -INFINITY ? 0.f : o2.y * ex2(o2.x - M));
      if (real && hh == 0 && !(L >= 1.f && L < INFINITY)) atomicOr(c.err, ERR_NONFINITE);
      const float iL = real && L > 0.f ? 1.f / L : 0.f;  // 0: rows that take no part
      const float fct = mx == -INFINITY ? 0.f : ex2(mx - M) * iL;
      pn = real ? ex2(xn - M) * iL : 0.f;
      // The exact probabilities: P in place of the logits (bf16 hi + lo, the
      // A operand of PV) and the candidates' column sums into the scores.
#pragma unroll
      for (int t = 0; t < kOwn; ++t) {
        const int i = 2 * t + hh;
        if (i < nch) {
          const bool pre = i < nPB;
          const int j16 = pre ? i : i - nPB;
          uint32_t hi[8], lo[8];
#pragma unroll
          for (int jj = 0; jj < 16; jj += 2) {
            // padding rows (garbage logits) contribute exact zeros
            const float p0 = real ? e[t][jj] * fct : 0.f;
            const float p1 = real ? e[t][jj + 1] * fct : 0.f;
            e[t][jj] = p0;
            e[t][jj + 1] = p1;
            const __nv_bfloat162 b = __floats2bfloat162_rn(p0, p1);
            hi[jj >> 1] = *reinterpret_cast<const uint32_t *>(&b);
            lo[jj >> 1] = pack_bf16(p0 - __low2float(b), p1 - __high2float(b));
          }
          const uint32_t cp = pre ? kColSP + 16 * j16 : col_t + 16 * j16;
          tmem_st8(trow + cp, hi);
          tmem_st8(trow + cp + 8, lo);
          const float2 cs = colsum8(e[t], r8);
          const int live = pre ? np : nt;
          const int key = 16 * j16 + 2 * r8;
          if (cand_ok && key < live) {  // one add per row and step: no read back
            float *dst = (pre ? ps : tsc) + key;
            atomicAdd(dst, cs.x * inv_g);
            if (key + 1 < live) atomicAdd(dst + 1, cs.y * inv_g);
          }
        }
      }
      tmem_wait_st();
    }
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_u32(&s.p_full[ts]));
    if (ok) {
      if (hh == 0) {  // the new row: its score, position and the tail length
        float sn = pn;
        sn += __shfl_xor_sync(0xffffffffu, sn, 4);
        sn += __shfl_xor_sync(0xffffffffu, sn, 2);
        sn += __shfl_xor_sync(0xffffffffu, sn, 1);
        if (cand_ok && r8 == 0) {
          tsc[nt] = sn * inv_g;
          f.tpos[cu * f.tstride + nt] = pos;
          f.tlen[cu] = nt + 1;
        }
      } else {  // append the new rows to the tails (from the head buffer)
        for (int i = par * 32 + lane; i < N * 32; i += 64) {
          const int cc = i >> 5, ch = i & 15;
          const bool v = (i & 16) != 0;
          const int4 val =
              *reinterpret_cast<const int4 *>(hd + (v ? Nv::vn : Nv::kn) + cc * 256 + ch * 16);
          const size_t cu2 = (size_t)cc * units + u.ug;
          __nv_bfloat16 *dst = reinterpret_cast<__nv_bfloat16 *>(v ? f.TV : f.TK) +
                               (cu2 * (size_t)f.tcap + nt) * 128;
          reinterpret_cast<int4 *>(dst)[ch] = val;
        }
      }
    }
    // ---- outputs: O (prefix and tail) + p_new * v_new ----
    alive = warp_wait(&s.o_full[ts], ph, s, c.err, kWaitNs);
    tc_fence_after();
    if (ok && alive) {
      float ov[4][16];
      const bool any = nch > 0;  // otherwise no MMA wrote O
      if (any) {
#pragma unroll
        for (int t = 0; t < 4; ++t) tmem_ld16f_nowait(trow + kColO + 64 * hh + 16 * t, ov[t]);
        tmem_wait_ld();
      }
      if (real) {
        const unsigned char *vnr = hd + Nv::vn + cand * 256 + 128 * hh;
        constexpr int osz = kOutBf16 ? 2 : 4;
        unsigned char *orow = reinterpret_cast<unsigned char *>(p.out) +
                              ((((size_t)cand * per + u.row0) * G + g) * 128 + 64 * hh) * osz;
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          float o[16];
          const uint4 va = *reinterpret_cast<const uint4 *>(vnr + 32 * t);
          const uint4 vb = *reinterpret_cast<const uint4 *>(vnr + 32 * t + 16);
          const uint32_t vv[8] = {va.x, va.y, va.z, va.w, vb.x, vb.y, vb.z, vb.w};
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const float2 v2 =
                __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&vv[j]));
            o[2 * j] = fmaf(pn, v2.x, any ? ov[t][2 * j] : 0.f);
            o[2 * j + 1] = fmaf(pn, v2.y, any ? ov[t][2 * j + 1] : 0.f);
          }
          if (kOutBf16) {
            uint32_t w[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) w[j] = pack_bf16(o[2 * j], o[2 * j + 1]);
            reinterpret_cast<int4 *>(orow + 32 * t)[0] = make_int4(w[0], w[1], w[2], w[3]);
            reinterpret_cast<int4 *>(orow + 32 * t)[1] = make_int4(w[4], w[5], w[6], w[7]);
          } else {
#pragma unroll
            for (int j = 0; j < 4; ++j)
              reinterpret_cast<float4 *>(orow + 64 * t)[j] =
                  make_float4(o[4 * j], o[4 * j + 1], o[4 * j + 2], o[4 * j + 3]);
          }
        }
      }
    }
    tc_fence_before();
    __syncwarp();
    if (lane == 0) {
      mbar_arrive(smem_u32(&s.o_free[ts]));
      mbar_arrive(smem_u32(&s.head_free[hb]));
    }
  }
}

template <bool kOutBf16, int kOwn>
__global__ void __launch_bounds__(kThreads, 1)
    fork_tc_kernel(const __grid_constant__ TcMaps maps, const ForkTcParams p) {
  extern __shared__ unsigned char smem_raw[];
  __shared__ Ctl s;
  unsigned char *smem = reinterpret_cast<unsigned char *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const CacheView &c = p.f.p;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_units = c.S * p.nl * c.H;
  const int mine = (int)blockIdx.x < n_units
                       ? (n_units - 1 - (int)blockIdx.x) / (int)gridDim.x + 1
                       : 0;
  if (warp == 1) tmem_alloc(smem_u32(&s.tmem), kTmemCols);
  if (threadIdx.x == 0) {
    prefetch_tmap(&maps.k);
    prefetch_tmap(&maps.v);
    prefetch_tmap(&maps.tk);
    prefetch_tmap(&maps.tv);
    for (int i = 0; i < kSlotsK; ++i) {
      mbar_init(smem_u32(&s.fullK[i]), 1);
      mbar_init(smem_u32(&s.emptyK[i]), 1);
    }
    for (int i = 0; i < kSlotsV; ++i) {
      mbar_init(smem_u32(&s.fullV[i]), 1);
      mbar_init(smem_u32(&s.emptyV[i]), 1);
    }
    for (int i = 0; i < kHeads; ++i) {
      mbar_init(smem_u32(&s.head_full[i]), 33);  // 32 cp.async lanes + header
      mbar_init(smem_u32(&s.head_free[i]), 4);   // the unit slot's 4 warps
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&s.q_free[i]), 4 + 1);  // the slot's 4 warps + S done
      mbar_init(smem_u32(&s.s_full[i]), 1);
      mbar_init(smem_u32(&s.p_full[i]), 4);
      mbar_init(smem_u32(&s.o_full[i]), 1);
      mbar_init(smem_u32(&s.o_free[i]), 4);
      mbar_init(smem_u32(&s.drain[i]), 1);
    }
    s.issuedK = s.consumedK = s.issuedV = s.consumedV = 0;
    s.abort = 0;
    fence_mbar_init();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_begin();

  if (warp == 0) {
    produce_k(p, maps, smem, s, mine, lane);
  } else if (warp == 1) {
    issue_s(p, smem, s, mine, lane);
  } else if (warp == 2) {
    issue_pv(p, smem, s, mine, lane);
  } else if (warp == 3) {
    produce_v(p, maps, smem, s, mine, lane);
  } else {
    softmax_epilogue<kOutBf16, kOwn>(p, smem, s, mine, warp, lane);
  }
  tc_fence_before();
  __syncthreads();
  // After an abort, wait (bounded) for copies still landing in the rings:
  // every item issued but not waited for by its issuer.
  if (s.abort && threadIdx.x == 0) {
    volatile int never = 0;
    for (int q = s.consumedK; q < s.issuedK; ++q) {
      const int e = s.logK[q % kSlotsK];
      mbar_wait(smem_u32(&s.fullK[e & 0xFF]), (uint32_t)(e >> 8) & 1u, &never);
    }
    for (int q = s.consumedV; q < s.issuedV; ++q) {
      const int e = s.logV[q % kSlotsV];
      mbar_wait(smem_u32(&s.fullV[e & 0xFF]), (uint32_t)(e >> 8) & 1u, &never);
    }
  }
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(s.tmem, kTmemCols);
}

}  // namespace

int fork_tc_max_cand() { return kMaxCand; }
int fork_tc_max_prefix() { return kMaxPrefix; }
int fork_tc_max_tail() { return kMaxTail; }
int fork_tc_box_rows() { return kBox; }
size_t fork_tc_smem_bytes() { return (size_t)Smem::alloc; }

cudaError_t launch_fork_tc(const CUtensorMap &tmK, const CUtensorMap &tmV,
                           const CUtensorMap *tmTK, const CUtensorMap *tmTV,
                           const ForkTcParams &p, int grid, cudaStream_t st) {
  if (p.f.N < 1 || p.f.N > kMaxCand || p.f.p.G > 8 || p.f.p.d != 128 ||
      !p.f.p.kv_bf16)
    return cudaErrorInvalidValue;
  TcMaps maps;
  maps.k = tmK;
  maps.v = tmV;
  maps.tk = *tmTK;
  maps.tv = *tmTV;
  // Chunks per unit at most: the prefix (np_max rows) and the tail.
  const int chunks = (p.np_max + 15) / 16 + (p.nt + 15) / 16;
  auto kern = chunks <= 10 ? (p.f.p.out_bf16 ? fork_tc_kernel<true, 5> : fork_tc_kernel<false, 5>)
                           : (p.f.p.out_bf16 ? fork_tc_kernel<true, 6> : fork_tc_kernel<false, 6>);
  cudaError_t e = cudaFuncSetAttribute(
      kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Smem::alloc);
  if (e != cudaSuccess) return e;
  return launch_pdl(kern, dim3(grid), dim3(kThreads), (size_t)Smem::alloc, st, maps, p);
}

}  // namespace kvr
