// kvr_fused_unit.cuh -- the per-unit body of the fused decode-step kernel
// (included by kvr_fused.cu only).
//
// One group of U warps computes one (sequence, layer, KV head) unit held in
// a shared-memory stage.  The unit has T = R / 16 row tiles; warp w of the
// group owns tiles w, w + U, ... and everything about their rows: inserting
// the new row if it falls in an owned tile, the logits, probabilities,
// accumulated-attention scores and eviction candidates.
//
// The work is split in two so that the stage is held only while its bytes
// are being read:
//  - unit_front (stage held): logits of the owned rows, their probabilities
//    relative to the warp's own per-head maximum, and the warp's partial
//    out^T = V^T P^T over its own rows for all 128 head-dim columns (the
//    split-softmax identity: partial outputs taken against local maxima
//    combine exactly once rescaled by exp2(local max - global max) / Z).
//    The stage is then released to the producer.
//  - unit_back (group-private memory only): one exchange of the per-head
//    (max, sum) statistics and the partial outputs, the merged output for
//    the warp's share of head-dim tiles, the accumulated-attention update of
//    the owned rows, and a second exchange to agree on the evicted row.
//
// Group exchange area (GroupLayout): XS, five 16-byte slots per warp (slot
// cp = 0..3 holds (max, max, sum, sum) of heads 2cp and 2cp + 1; slot 4
// holds the warp's eviction candidate (key low, key high, row, 0)), and OX,
// the warps' partial outputs as [warp][head-dim tile][lane] float4s.

template <int TW>
struct UnitFront {
  size_t ug;    // cache unit
  size_t krow;  // row of this unit in the call's [S][nl][H] inputs
  int m, t;     // live rows before the append; position of the new row
  bool own_new; // this warp owns the tile of row m
  float pr[TW][4];          // exp2(logit - warp max) of the owned rows
  float ref0, ref1, z0, z1; // warp max and sum per head (columns c2, c2+1)
  float o[8][4];            // partial out^T, head-dim tiles 0..7
  float sc[TW][2];          // old scores of rows r0 and r0 + 8 of each tile
  int ps[TW][2];            // their positions
  int4 nrow;                // own_new warp: 16 bytes of the new k (lanes
                            // 0-15) or v (lanes 16-31) row
  float rr[TW][2];          // R-KV step: mean cosine of rows r0, r0 + 8
                            // with the other live rows
  float s4[4];              // R-KV step, the warp owning the new row: the
                            // key sum after the append, dims 4 lane .. + 3
};

// 1 / |k| of one key held as four dims a lane (0 for a zero key); every
// lane gets the same value.  The library's kept key sum adds and removes a
// row's normalised key with this same arithmetic.
__device__ __forceinline__ float warp_inv_norm(const float (&k)[4]) {
  float ss = fmaf(k[3], k[3], fmaf(k[2], k[2], fmaf(k[1], k[1], k[0] * k[0])));
  ss = dev::warp_sum(ss);
  return ss > 0.f ? rsqrtf(ss) : 0.f;
}

// x as three bf16 terms t[0] + t[1] + t[2] (the third rounded when packed).
__device__ __forceinline__ void split3(float x, float (&t)[3]) {
  const float h = __bfloat162float(__float2bfloat16_rn(x));
  const float r = x - h;
  const float m = __bfloat162float(__float2bfloat16_rn(r));
  t[0] = h;
  t[1] = m;
  t[2] = r - m;
}

// The key sum S as the B operand of K S (m16n8k16; columns 0-2 the three
// terms of S): lane 4 t + p holds term t of dims 16 ks + 2 p, + 1 (word 0)
// and 16 ks + 8 + 2 p, + 1 (word 1).  Each lane holds S for dims
// 4 lane .. + 3 in s4; the terms pass through this warp's scratch sbx
// ([8][12][2] words) in that order.
__device__ __forceinline__ void key_sum_fragments(const float (&s4)[4],
                                                  uint32_t *sbx, int lane,
                                                  uint32_t (&sb)[8][2]) {
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int d = 4 * lane + 2 * h;
    const int ks = d >> 4, j = d & 15, reg = j >> 3, pp = (j & 7) >> 1;
    float a[3], b[3];
    split3(s4[2 * h], a);
    split3(s4[2 * h + 1], b);
#pragma unroll
    for (int t = 0; t < 3; ++t)
      sbx[(ks * 12 + 4 * t + pp) * 2 + reg] = pack_bf16(a[t], b[t]);
  }
  __syncwarp();
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    if (lane < 12) {
      const uint2 v = *reinterpret_cast<const uint2 *>(sbx + (ks * 12 + lane) * 2);
      sb[ks][0] = v.x;
      sb[ks][1] = v.y;
    } else {
      sb[ks][0] = sb[ks][1] = 0u;
    }
  }
}

// Dims 4 lane .. 4 lane + 3 of a bf16 row of 128.
__device__ __forceinline__ void row4(const void *row, int lane, float (&k)[4]) {
  const uint2 w = *reinterpret_cast<const uint2 *>(
      static_cast<const unsigned char *>(row) + 8 * lane);
  k[0] = __uint_as_float(w.x << 16);
  k[1] = __uint_as_float(w.x & 0xffff0000u);
  k[2] = __uint_as_float(w.y << 16);
  k[3] = __uint_as_float(w.y & 0xffff0000u);
}

// x as three bf16 terms (x0 + x1 + x2 carries the 24-bit mantissa): term t.
__device__ __forceinline__ float bf16_term(float x, int t) {
  const float h = __bfloat162float(__float2bfloat16_rn(x));
  if (t == 0) return h;
  const float m = __bfloat162float(__float2bfloat16_rn(x - h));
  return t == 1 ? m : x - h - m;
}

template <int T, int U, bool kRkv>
__device__ __forceinline__ bool unit_front(const FusedParams &p,
                                           unsigned char *stage, int idx,
                                           int w, int lane,
                                           UnitFront<(T + U - 1) / U> &f,
                                           unsigned char *garea, int bar_id) {
  constexpr int TW = (T + U - 1) / U;  // tiles per warp (at most)
  constexpr int R = 16 * T;
  const StageLayout L(R, kRkv);
  {
    const UnitIdx x = unit_idx(p, idx);
    f.ug = x.ug;
    f.krow = x.krow;
  }
  unsigned char *K0 = stage + L.k0, *K1 = stage + L.k1;
  unsigned char *V0 = stage + L.v0, *V1 = stage + L.v1;
  const unsigned char *KN = stage + L.kn, *VN = stage + L.vn;
  const float *SC = reinterpret_cast<const float *>(stage + L.sc);
  const int32_t *PS = reinterpret_cast<const int32_t *>(stage + L.ps);
  const int32_t *ST = reinterpret_cast<const int32_t *>(stage + L.st);
  f.m = ST[0];
  f.t = ST[1];
  const int m = f.m, n = m + 1;
  if (m < 0 || n > R) {  // same decision in every warp of the group
    if (w == 0 && lane == 0) atomicOr(p.c.err, ERR_LENGTH);
    return false;
  }
  f.own_new = ((m >> 4) % U) == w;

  // 1. Insert the new row as logical row m (swizzled like the TMA boxes) and
  //    zero V beyond it in the owned tiles, so padded rows contribute 0.
  if (f.own_new) {
    const int chunk = lane & 15, half = chunk >> 3, cc = chunk & 7;
    const uint32_t off = m * 128 + ((cc ^ (m & 7)) << 4);
    unsigned char *dst = lane < 16 ? (half ? K1 : K0) : (half ? V1 : V0);
    const unsigned char *src = lane < 16 ? KN : VN;
    f.nrow = *reinterpret_cast<const int4 *>(src + chunk * 16);
    *reinterpret_cast<int4 *>(dst + off) = f.nrow;
  }
#pragma unroll
  for (int j = 0; j < TW; ++j) {
    const int tt = w + j * U;
    const int r_lo = max(tt * 16, m + 1), r_hi = tt * 16 + 16;
    if (tt < T && r_lo < r_hi)
      for (int i = lane; i < (r_hi - r_lo) * 16; i += 32) {
        const int r = r_lo + (i >> 4), c16 = i & 15;
        *reinterpret_cast<int4 *>((c16 < 8 ? V0 : V1) + r * 128 +
                                  (c16 & 7) * 16) = make_int4(0, 0, 0, 0);
        // A fresh R-KV key sum reads every row of the tile: padding keys
        // must be zeros too (rows past the box are stale).
        if (kRkv && ST[2] != 1)
          *reinterpret_cast<int4 *>((c16 < 8 ? K0 : K1) + r * 128 +
                                    (c16 & 7) * 16) = make_int4(0, 0, 0, 0);
      }
  }
  __syncwarp();

  // 2. Query heads as the MMA B operand (k = head dim, n = query head).
  uint32_t qb[8][2];
  {
    const uint32_t qa = smem_u32(stage + L.q) + (lane & 7) * kQPitch +
                        (lane >> 3) * 16;
#pragma unroll
    for (int i = 0; i < 4; ++i)
      ldsm_x4(qa + i * 64, qb[2 * i][0], qb[2 * i][1], qb[2 * i + 1][0],
              qb[2 * i + 1][1]);
  }

  // 3. Logits of the owned tiles: m16n8 per 16 rows, 8 k-steps split over
  //    two accumulator chains.  The R-KV step also takes the tile's Gram
  //    blocks K K^T from the same A fragments (K rows are a row-major B
  //    operand as they stand): their diagonals are the squared key norms,
  //    and inv holds 1 / |k| of rows r0 and r0 + 8 (0 for a zero key and
  //    for rows past the live ones).
  float (&acc)[TW][4] = f.pr;
  float inv[TW][2];
#pragma unroll
  for (int j = 0; j < TW; ++j) {
    float a2[4] = {0.f, 0.f, 0.f, 0.f};
    float g0[4] = {0.f, 0.f, 0.f, 0.f}, g1[4] = {0.f, 0.f, 0.f, 0.f};
    acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;
    inv[j][0] = inv[j][1] = 0.f;
    const int tt = w + j * U;
    if (tt < T) {
      const int row = tt * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
      const uint32_t b0 = smem_u32(K0) + row * 128, b1 = smem_u32(K1) + row * 128;
#pragma unroll
      for (int ks = 0; ks < 8; ++ks) {
        const int cc = ((ks & 3) << 1) + (lane >> 4);
        const uint32_t addr = (ks >> 2 ? b1 : b0) + ((cc ^ (row & 7)) << 4);
        uint32_t a0, a1, a2r, a3;
        ldsm_x4(addr, a0, a1, a2r, a3);
        if (ks & 1)
          mma_bf16(a2, a0, a1, a2r, a3, qb[ks][0], qb[ks][1]);
        else
          mma_bf16(acc[j], a0, a1, a2r, a3, qb[ks][0], qb[ks][1]);
        if constexpr (kRkv) {
          mma_bf16(g0, a0, a1, a2r, a3, a0, a2r);  // columns: rows 0-7
          mma_bf16(g1, a0, a1, a2r, a3, a1, a3);   // columns: rows 8-15
        }
      }
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[j][e] += a2[e];
      if constexpr (kRkv) {
        // Diagonal (r, r) of a block sits in lane 4 r + r / 2, register
        // r & 1 (rows 0-7) or 2 + (r & 1) (rows 8-15).
        const int rl = lane >> 2;
        const float x = (rl & 1) ? g0[1] : g0[0];
        const float y = (rl & 1) ? g1[3] : g1[2];
        const int src = 4 * rl + (rl >> 1);
        const float na = __shfl_sync(0xffffffffu, x, src);
        const float nb = __shfl_sync(0xffffffffu, y, src);
        const int ra = tt * 16 + rl, rb = ra + 8;
        inv[j][0] = (ra < n && na > 0.f) ? rsqrtf(na) : 0.f;
        inv[j][1] = (rb < n && nb > 0.f) ? rsqrtf(nb) : 0.f;
      }
    }
  }

  if constexpr (kRkv) {
    // 3b. R-KV redundancy (App. C, the library's reading): r_i, the mean
    //     cosine of key i with the other n - 1 live keys, is
    //     (k_i . S / |k_i| - 1) / (n - 1) with S the sum of the normalised
    //     live keys (no n x n similarity).  Both products run on the tensor
    //     cores with the fp32 vector split into three bf16 terms (columns
    //     0-2 of the B operand; their sum carries the full mantissa):
    //     S^T = K^T (1/|k|) in the PV product's form, then K S.
    const int c2 = (lane & 3) * 2, rl = lane >> 2;
    float *SX = reinterpret_cast<float *>(garea + GroupLayout(U, true).ox);
    const float *RS = reinterpret_cast<const float *>(stage + L.rs);
    // A kept sum (state word 2 set by the previous R-KV step of this unit)
    // needs only the new key added: S = kept + k_new / |k_new|.  Otherwise
    // the group sums every live row's normalised key afresh.
    const bool warm = ST[2] == 1;
    uint32_t sb[8][2];
    if (warm) {
      float kn4[4], s4[4];
      row4(KN, lane, kn4);
      const float inv_new = warp_inv_norm(kn4);
      const float4 rs = reinterpret_cast<const float4 *>(RS)[lane];
      s4[0] = fmaf(kn4[0], inv_new, rs.x);
      s4[1] = fmaf(kn4[1], inv_new, rs.y);
      s4[2] = fmaf(kn4[2], inv_new, rs.z);
      s4[3] = fmaf(kn4[3], inv_new, rs.w);
      // This warp's own partial-output slot is free until unit_publish.
      key_sum_fragments(s4, reinterpret_cast<uint32_t *>(SX) + w * 1024, lane,
                        sb);
      if (f.own_new)
#pragma unroll
        for (int e = 0; e < 4; ++e) f.s4[e] = s4[e];
    } else {
      float fs[8][4];
#pragma unroll
      for (int i = 0; i < 8; ++i) fs[i][0] = fs[i][1] = fs[i][2] = fs[i][3] = 0.f;
#pragma unroll
      for (int j = 0; j < TW; ++j) {
        const int tt = w + j * U;
        if (tt >= T) continue;
        // Columns (c2, c2 + 1) of rows r0 and r0 + 8: terms 0, 1 in lanes
        // c2 = 0, term 2 in lanes c2 = 2.
        const float ia = inv[j][0], ib = inv[j][1];
        const uint32_t h0 =
            c2 == 0 ? pack_bf16(bf16_term(ia, 0), bf16_term(ia, 1))
                    : (c2 == 2 ? pack_bf16(bf16_term(ia, 2), 0.f) : 0u);
        const uint32_t h1 =
            c2 == 0 ? pack_bf16(bf16_term(ib, 0), bf16_term(ib, 1))
                    : (c2 == 2 ? pack_bf16(bf16_term(ib, 2), 0.f) : 0u);
        const uint32_t pb0 = movm_t(h0), pb1 = movm_t(h1);
        const int row = tt * 16 + (lane & 7) + ((lane >> 4) << 3);
        const uint32_t b0 = smem_u32(K0) + row * 128, b1 = smem_u32(K1) + row * 128;
#pragma unroll
        for (int mt = 0; mt < 8; ++mt) {
          const int c16 = 2 * mt + ((lane >> 3) & 1);
          const uint32_t addr = (c16 >> 3 ? b1 : b0) + (((c16 & 7) ^ (row & 7)) << 4);
          uint32_t a0, a1, a2, a3;
          ldsm_x4_t(addr, a0, a1, a2, a3);
          mma_bf16(fs[mt], a0, a1, a2, a3, pb0, pb1);
        }
      }
      // This warp's part of S, dims mt * 16 + r0 (+ 8): columns 0 + 1 in
      // the lane with c2 = 0, column 2 one lane up.
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) {
        const float t2a = __shfl_down_sync(0xffffffffu, fs[mt][0], 1);
        const float t2b = __shfl_down_sync(0xffffffffu, fs[mt][2], 1);
        if (c2 == 0) {
          SX[w * 128 + mt * 16 + rl] = fs[mt][0] + fs[mt][1] + t2a;
          SX[w * 128 + mt * 16 + rl + 8] = fs[mt][2] + fs[mt][3] + t2b;
        }
      }
      group_bar(bar_id, 32 * U);
      // S as the dots' B operand (as above); the warps' parts are added in
      // warp order.
#pragma unroll
      for (int ks = 0; ks < 8; ++ks) {
        float v[4] = {0.f, 0.f, 0.f, 0.f};
        if (lane < 12) {
          const int d0 = 16 * ks + 2 * (lane & 3);
#pragma unroll
          for (int u = 0; u < U; ++u) {
            v[0] += SX[u * 128 + d0];
            v[1] += SX[u * 128 + d0 + 1];
            v[2] += SX[u * 128 + d0 + 8];
            v[3] += SX[u * 128 + d0 + 9];
          }
          const int t = lane >> 2;
#pragma unroll
          for (int e = 0; e < 4; ++e) v[e] = bf16_term(v[e], t);
        }
        sb[ks][0] = pack_bf16(v[0], v[1]);
        sb[ks][1] = pack_bf16(v[2], v[3]);
      }
      if (f.own_new)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          float x = 0.f;
#pragma unroll
          for (int u = 0; u < U; ++u) x += SX[u * 128 + 4 * lane + e];
          f.s4[e] = x;
        }
      // Every warp has read the parts before any writes the area again
      // (unit_publish).
      group_bar(bar_id, 32 * U);
    }
    const float inv_n1 = n > 1 ? 1.f / (float)(n - 1) : 0.f;
#pragma unroll
    for (int j = 0; j < TW; ++j) {
      f.rr[j][0] = f.rr[j][1] = 0.f;
      const int tt = w + j * U;
      if (tt >= T) continue;
      float dd[4] = {0.f, 0.f, 0.f, 0.f};
      const int row = tt * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
      const uint32_t b0 = smem_u32(K0) + row * 128, b1 = smem_u32(K1) + row * 128;
#pragma unroll
      for (int ks = 0; ks < 8; ++ks) {
        const int cc = ((ks & 3) << 1) + (lane >> 4);
        const uint32_t addr = (ks >> 2 ? b1 : b0) + ((cc ^ (row & 7)) << 4);
        uint32_t a0, a1, a2r, a3;
        ldsm_x4(addr, a0, a1, a2r, a3);
        mma_bf16(dd, a0, a1, a2r, a3, sb[ks][0], sb[ks][1]);
      }
      const float t2a = __shfl_down_sync(0xffffffffu, dd[0], 1);
      const float t2b = __shfl_down_sync(0xffffffffu, dd[2], 1);
      float da = dd[0] + dd[1] + t2a, db = dd[2] + dd[3] + t2b;
      da = __shfl_sync(0xffffffffu, da, lane & ~3);
      db = __shfl_sync(0xffffffffu, db, lane & ~3);
      f.rr[j][0] = (da * inv[j][0] - (inv[j][0] > 0.f ? 1.f : 0.f)) * inv_n1;
      f.rr[j][1] = (db * inv[j][1] - (inv[j][1] > 0.f ? 1.f : 0.f)) * inv_n1;
    }
  }

  // 4. Probabilities relative to the warp's own maximum per query head
  //    (this lane holds heads c2 and c2 + 1); rows >= n are masked.
  const int r0 = lane >> 2;
  float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
  for (int j = 0; j < TW; ++j) {
    const int ra = (w + j * U) * 16 + r0, rb = ra + 8;
    acc[j][0] = ra < n ? acc[j][0] * p.scale_log2e : -INFINITY;
    acc[j][1] = ra < n ? acc[j][1] * p.scale_log2e : -INFINITY;
    acc[j][2] = rb < n ? acc[j][2] * p.scale_log2e : -INFINITY;
    acc[j][3] = rb < n ? acc[j][3] * p.scale_log2e : -INFINITY;
    mx0 = fmaxf(mx0, fmaxf(acc[j][0], acc[j][2]));
    mx1 = fmaxf(mx1, fmaxf(acc[j][1], acc[j][3]));
  }
#pragma unroll
  for (int o = 4; o < 32; o <<= 1) {
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, o));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, o));
  }
  // A warp whose rows are all padding has max -inf: use 0 as its reference
  // so that exp2(-inf - 0) = 0 instead of NaN.
  f.ref0 = mx0 == -INFINITY ? 0.f : mx0;
  f.ref1 = mx1 == -INFINITY ? 0.f : mx1;
  float z0 = 0.f, z1 = 0.f;
#pragma unroll
  for (int j = 0; j < TW; ++j) {
    acc[j][0] = ex2(acc[j][0] - f.ref0);
    acc[j][1] = ex2(acc[j][1] - f.ref1);
    acc[j][2] = ex2(acc[j][2] - f.ref0);
    acc[j][3] = ex2(acc[j][3] - f.ref1);
    z0 += acc[j][0] + acc[j][2];
    z1 += acc[j][1] + acc[j][3];
  }
#pragma unroll
  for (int o = 4; o < 32; o <<= 1) {
    z0 += __shfl_xor_sync(0xffffffffu, z0, o);
    z1 += __shfl_xor_sync(0xffffffffu, z1, o);
  }
  f.z0 = z0;
  f.z1 = z1;

  // 5. Old scores and positions of the owned rows (the new row m has score
  //    0 and position t).
#pragma unroll
  for (int j = 0; j < TW; ++j)
#pragma unroll
    for (int hsel = 0; hsel < 2; ++hsel) {
      const int r = (w + j * U) * 16 + r0 + 8 * hsel;
      f.sc[j][hsel] = r < m ? SC[r] : 0.f;
      f.ps[j][hsel] = r < m ? PS[r] : f.t;
    }

  // 6. Partial out^T = V^T P^T over the owned row tiles for every head-dim
  //    tile: M = head dim, K = rows, N = query heads.  P enters as two bf16
  //    terms (hi + lo carries ~16 mantissa bits; one bf16 term would cost up
  //    to 2^-9 relative per probability), each 8x8 block transposed in
  //    registers into the B operand layout.
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int e = 0; e < 4; ++e) f.o[i][e] = 0.f;
#pragma unroll
  for (int j = 0; j < TW; ++j) {
    const int tt = w + j * U;
    if (tt >= T) continue;
    const uint32_t h0 = pack_bf16(acc[j][0], acc[j][1]);
    const uint32_t h1 = pack_bf16(acc[j][2], acc[j][3]);
    const __nv_bfloat162 hb0 = *reinterpret_cast<const __nv_bfloat162 *>(&h0);
    const __nv_bfloat162 hb1 = *reinterpret_cast<const __nv_bfloat162 *>(&h1);
    const uint32_t l0 = pack_bf16(acc[j][0] - __low2float(hb0),
                                  acc[j][1] - __high2float(hb0));
    const uint32_t l1 = pack_bf16(acc[j][2] - __low2float(hb1),
                                  acc[j][3] - __high2float(hb1));
    const uint32_t ph0 = movm_t(h0), ph1 = movm_t(h1);
    const uint32_t pl0 = movm_t(l0), pl1 = movm_t(l1);
    const int row = tt * 16 + (lane & 7) + ((lane >> 4) << 3);
    const uint32_t b0 = smem_u32(V0) + row * 128, b1 = smem_u32(V1) + row * 128;
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) {
      const int c16 = 2 * mt + ((lane >> 3) & 1);
      const uint32_t addr = (c16 >> 3 ? b1 : b0) + (((c16 & 7) ^ (row & 7)) << 4);
      uint32_t a0, a1, a2, a3;
      ldsm_x4_t(addr, a0, a1, a2, a3);
      mma_bf16(f.o[mt], a0, a1, a2, a3, ph0, ph1);
      mma_bf16(f.o[mt], a0, a1, a2, a3, pl0, pl1);
    }
  }
  return true;
}

// The warp's statistics and partial output into the group area (U > 1);
// after this the partial-output registers are free.
template <int T, int U, bool kRkv>
__device__ __forceinline__ void unit_publish(unsigned char *garea,
                                             const UnitFront<(T + U - 1) / U> &f,
                                             int w, int lane) {
  if constexpr (U > 1) {
    const GroupLayout GL(U, kRkv);
    float4 *XS4 = reinterpret_cast<float4 *>(garea + GL.xs);
    float4 *OX = reinterpret_cast<float4 *>(garea + GL.ox);
    if (lane < 4)
      XS4[w * GL.slots + lane] = make_float4(f.ref0, f.ref1, f.z0, f.z1);
#pragma unroll
    for (int mt = 0; mt < 8; ++mt)
      OX[(w * 8 + mt) * 32 + lane] =
          make_float4(f.o[mt][0], f.o[mt][1], f.o[mt][2], f.o[mt][3]);
  }
}

constexpr float kLog2e = 1.4426950408889634f;

template <int T, int U, bool kOutBf16, bool kRkv>
__device__ __forceinline__ void unit_back(const FusedParams &p,
                                          unsigned char *garea,
                                          UnitFront<(T + U - 1) / U> &f,
                                          int w, int lane, int bar_id) {
  constexpr int TW = (T + U - 1) / U;
  const GroupLayout GL(U, kRkv);
  const int G = p.c.G;
  const int m = f.m, n = m + 1, t = f.t;
  const int r0 = lane >> 2, c2 = (lane & 3) * 2;
  float4 *XS4 = reinterpret_cast<float4 *>(garea + GL.xs);
  float4 *OX = reinterpret_cast<float4 *>(garea + GL.ox);

  // 7. Merge the published statistics (unit_publish).  fv0[v] and fv1[v]
  //    rescale warp v's terms of heads c2 and c2 + 1: exp2(max_v - max) / Z.
  //    Warps with no live row (sum 0) take no part.
  float fv0[U], fv1[U];
  float Z0, Z1;
  if constexpr (U > 1) {
    group_bar(bar_id, 32 * U);
    float4 r[U];
    float M0 = -INFINITY, M1 = -INFINITY;
#pragma unroll
    for (int v = 0; v < U; ++v) {
      r[v] = XS4[v * GL.slots + (lane & 3)];
      if (r[v].z > 0.f) M0 = fmaxf(M0, r[v].x);
      if (r[v].w > 0.f) M1 = fmaxf(M1, r[v].y);
    }
    float S0 = 0.f, S1 = 0.f;
#pragma unroll
    for (int v = 0; v < U; ++v) {
      fv0[v] = r[v].z > 0.f ? ex2(r[v].x - M0) : 0.f;
      fv1[v] = r[v].w > 0.f ? ex2(r[v].y - M1) : 0.f;
      S0 += r[v].z * fv0[v];
      S1 += r[v].w * fv1[v];
    }
    const float i0 = rcp(S0), i1 = rcp(S1);
#pragma unroll
    for (int v = 0; v < U; ++v) {
      fv0[v] *= i0;
      fv1[v] *= i1;
    }
    Z0 = S0;  // >= 1: the warp holding the maximum contributes exp2(0)
    Z1 = S1;
  } else {
    fv0[0] = rcp(f.z0);
    fv1[0] = rcp(f.z1);
    Z0 = f.z0;
    Z1 = f.z1;
  }
  // Lanes 0-3 hold the sums of all eight heads (2 each); a NaN or an
  // infinity in q, k or the scale leaves one of them non-finite.
  if (w == 0 && lane < 4 &&
      !(Z0 > 0.5f && Z0 < INFINITY && Z1 > 0.5f && Z1 < INFINITY))
    atomicOr(p.c.err, ERR_NONFINITE);
  float f0 = fv0[0], f1 = fv1[0];
#pragma unroll
  for (int v = 1; v < U; ++v)
    if (v == w) {
      f0 = fv0[v];
      f1 = fv1[v];
    }

  // 8. Output tiles this warp owns (head-dim tiles mt = w, w + U, ...):
  //    the rescaled sum of every warp's partial, stored from the fragments.
  {
    constexpr int MW = (8 + U - 1) / U;
    constexpr int osz = kOutBf16 ? 2 : 4;
    unsigned char *gout = reinterpret_cast<unsigned char *>(p.out) +
                          f.krow * G * 128 * osz;
#pragma unroll
    for (int i = 0; i < MW; ++i) {
      const int mt = w + i * U;
      if (mt >= 8) continue;
      float e0 = 0.f, e1 = 0.f, e2 = 0.f, e3 = 0.f;
      if constexpr (U > 1) {
#pragma unroll
        for (int v = 0; v < U; ++v) {
          const float4 x = OX[(v * 8 + mt) * 32 + lane];
          e0 += x.x * fv0[v];
          e1 += x.y * fv1[v];
          e2 += x.z * fv0[v];
          e3 += x.w * fv1[v];
        }
      } else {
        e0 = f.o[mt][0] * f0;
        e1 = f.o[mt][1] * f1;
        e2 = f.o[mt][2] * f0;
        e3 = f.o[mt][3] * f1;
      }
      if (kOutBf16) {
        // (head dim, head) 8x8 blocks -> (head, head dim) pairs per lane.
        const uint32_t lo = movm_t(pack_bf16(e0, e1));
        const uint32_t hi = movm_t(pack_bf16(e2, e3));
        const int g = lane >> 2, dd = 16 * mt + 2 * (lane & 3);
        if (g < G) {
          *reinterpret_cast<uint32_t *>(gout + ((size_t)g * 128 + dd) * 2) = lo;
          *reinterpret_cast<uint32_t *>(gout + ((size_t)g * 128 + dd + 8) * 2) = hi;
        }
      } else {
        float *of = reinterpret_cast<float *>(gout);
        const int d0 = 16 * mt + r0;
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

  // 9. Accumulated attention of the owned rows (score += mean over the G
  //    heads of the normalised probability), written back at once except
  //    for the new row; the warp's eviction candidate (lowest
  //    (score, -position) outside the window).
  const bool g0 = c2 < G, g1 = c2 + 1 < G;
  const int wlo = t - p.window;  // a row is a candidate iff pos <= wlo
  float *gsc = p.c.score + f.ug * p.c.sstride;
  unsigned long long best = ~0ull;
  int bi = -1;
  float new_score = 0.f;
  float sv[TW][2];  // R-KV step: updated scores of the owned rows
#pragma unroll
  for (int j = 0; j < TW; ++j) {
    sv[j][0] = sv[j][1] = 0.f;
    float sa = (g0 ? f.pr[j][0] * f0 : 0.f) + (g1 ? f.pr[j][1] * f1 : 0.f);
    float sb = (g0 ? f.pr[j][2] * f0 : 0.f) + (g1 ? f.pr[j][3] * f1 : 0.f);
    sa += __shfl_xor_sync(0xffffffffu, sa, 1);
    sb += __shfl_xor_sync(0xffffffffu, sb, 1);
    sa += __shfl_xor_sync(0xffffffffu, sa, 2);
    sb += __shfl_xor_sync(0xffffffffu, sb, 2);
    const int tt = w + j * U;
    if ((lane & 3) == 0 && tt < T) {
#pragma unroll
      for (int hsel = 0; hsel < 2; ++hsel) {
        const int r = tt * 16 + r0 + 8 * hsel;
        if (r < n) {
          const float s = f.sc[j][hsel] + (hsel ? sb : sa) * p.inv_g;
          if (r < m) gsc[r] = s;
          else new_score = s;
          sv[j][hsel] = s;
          const int pr = f.ps[j][hsel];
          if (!kRkv && pr <= wlo) {
            const unsigned long long key =
                ((unsigned long long)__float_as_uint(s) << 32) |
                (unsigned long long)(0xFFFFFFFFu - (unsigned)pr);
            if (key < best) {
              best = key;
              bi = r;
            }
          }
        }
      }
    }
  }
  // The lane that scored the new row passes its score to the whole warp.
  new_score = __shfl_sync(0xffffffffu, new_score, ((m & 15) & 7) * 4);
  if constexpr (kRkv) {
    // R-KV (App. C, the library's reading) over the candidates C (rows
    // outside the window): I = s / sum_C s, R = softmax_C(r) and
    // z = lam I - (1 - lam) R; the victim is the lowest (z, -position).
    // Each warp reduces its own candidates (sum of s, max of r and the
    // sum of exp(r - max)); the group merges them in warp order.
    float ssum = 0.f, rmax = -INFINITY;
#pragma unroll
    for (int j = 0; j < TW; ++j)
#pragma unroll
      for (int hsel = 0; hsel < 2; ++hsel) {
        const int r = (w + j * U) * 16 + r0 + 8 * hsel;
        if ((lane & 3) == 0 && w + j * U < T && r < n &&
            f.ps[j][hsel] <= wlo) {
          ssum += sv[j][hsel];
          rmax = fmaxf(rmax, f.rr[j][hsel]);
        }
      }
    ssum = dev::warp_sum(ssum);
    rmax = dev::warp_max(rmax);
    float esum = 0.f;
#pragma unroll
    for (int j = 0; j < TW; ++j)
#pragma unroll
      for (int hsel = 0; hsel < 2; ++hsel) {
        const int r = (w + j * U) * 16 + r0 + 8 * hsel;
        if ((lane & 3) == 0 && w + j * U < T && r < n &&
            f.ps[j][hsel] <= wlo)
          esum += ex2((f.rr[j][hsel] - rmax) * kLog2e);
      }
    esum = dev::warp_sum(esum);
    float Ssum = ssum, M = rmax, E = esum;
    if constexpr (U > 1) {
      if (lane == 0) XS4[w * GL.slots + 5] = make_float4(ssum, rmax, esum, 0.f);
      group_bar(bar_id, 32 * U);
      Ssum = 0.f;
      M = -INFINITY;
#pragma unroll
      for (int v = 0; v < U; ++v) {
        const float4 x = XS4[v * GL.slots + 5];
        Ssum += x.x;
        if (x.z > 0.f) M = fmaxf(M, x.y);
      }
      E = 0.f;
#pragma unroll
      for (int v = 0; v < U; ++v) {
        const float4 x = XS4[v * GL.slots + 5];
        if (x.z > 0.f) E += x.z * ex2((x.y - M) * kLog2e);
      }
    }
    const float inv_s = Ssum > 0.f ? 1.f / Ssum : 0.f;
    const float inv_e = E > 0.f ? 1.f / E : 0.f;
#pragma unroll
    for (int j = 0; j < TW; ++j)
#pragma unroll
      for (int hsel = 0; hsel < 2; ++hsel) {
        const int r = (w + j * U) * 16 + r0 + 8 * hsel;
        const int pr = f.ps[j][hsel];
        if ((lane & 3) == 0 && w + j * U < T && r < n && pr <= wlo) {
          const float z = p.lam * (sv[j][hsel] * inv_s) -
                          (1.f - p.lam) *
                              (ex2((f.rr[j][hsel] - M) * kLog2e) * inv_e);
          const unsigned long long key = dev::rkv_key(z, pr);
          if (key < best) {
            best = key;
            bi = r;
          }
        }
      }
  }
  {
    // Warp argmin of the key: lowest score bits, then highest position
    // (keys are distinct because positions are).
    const uint32_t sb = bi < 0 ? 0xFFFFFFFFu : (uint32_t)(best >> 32);
    const int pb = bi < 0 ? -1 : (int)(0xFFFFFFFFu - (uint32_t)best);
    const uint32_t smin = __reduce_min_sync(0xffffffffu, sb);
    const int pmax = __reduce_max_sync(0xffffffffu, sb == smin ? pb : -1);
    const uint32_t who = __ballot_sync(0xffffffffu, bi >= 0 && sb == smin && pb == pmax);
    if (who) {
      bi = __shfl_sync(0xffffffffu, bi, __ffs(who) - 1);
      best = ((unsigned long long)smin << 32) |
             (unsigned long long)(0xFFFFFFFFu - (uint32_t)pmax);
    } else {
      bi = -1;
      best = ~0ull;
    }
  }

  // 10. Agree on the group's candidate.
  if constexpr (U > 1) {
    uint4 *XW = reinterpret_cast<uint4 *>(XS4);
    if (lane == 0)
      XW[w * GL.slots + 4] = make_uint4((uint32_t)best, (uint32_t)(best >> 32),
                                        (uint32_t)bi, 0u);
    group_bar(bar_id, 32 * U);
#pragma unroll
    for (int v = 0; v < U; ++v) {
      const uint4 a = XW[v * GL.slots + 4];
      const unsigned long long kb = ((unsigned long long)a.y << 32) | a.x;
      if (kb < best) {
        best = kb;
        bi = (int)a.z;
      }
    }
  }

  // 11. The warp owning the new row writes it into the freed slot (or the
  //     first free slot when nothing is evicted), with its position, score,
  //     the live length and the next position.
  if (f.own_new) {
    const int victim = (p.evict && n > p.budget + p.window) ? bi : -1;
    const int slot = victim < 0 ? m : (victim < m ? victim : -1);
    if constexpr (kRkv) {
      // The kept key sum after the step: the evicted row's normalised key
      // (from the slab, or the new row's own when it is the one evicted)
      // comes out, read before the new row overwrites its slot.
      if (victim >= 0) {
        float kv[4];
        row4(victim < m ? reinterpret_cast<const unsigned char *>(p.c.K) +
                              (f.ug * (size_t)p.c.cap + victim) * 256
                        : reinterpret_cast<const unsigned char *>(p.k_new) +
                              f.krow * 256,
             lane, kv);
        const float iv = warp_inv_norm(kv);
#pragma unroll
        for (int e = 0; e < 4; ++e) f.s4[e] = fmaf(-kv[e], iv, f.s4[e]);
      }
      *reinterpret_cast<float4 *>(p.c.rsum + f.ug * 128 + 4 * lane) =
          make_float4(f.s4[0], f.s4[1], f.s4[2], f.s4[3]);
      __syncwarp();
    }
    if (slot >= 0) {
      const int chunk = lane & 15;
      __nv_bfloat16 *dst =
          reinterpret_cast<__nv_bfloat16 *>(lane < 16 ? p.c.K : p.c.V) +
          (f.ug * (size_t)p.c.cap + slot) * 128;
      reinterpret_cast<int4 *>(dst)[chunk] = f.nrow;
      if (lane == 0) {
        p.c.pos[f.ug * p.c.sstride + slot] = t;
        gsc[slot] = new_score;
      }
    }
    if (lane == 0) {
      p.c.state[4 * f.ug] = victim < 0 ? m + 1 : m;
      p.c.state[4 * f.ug + 1] = t + 1;
      p.c.state[4 * f.ug + 2] = kRkv ? 1 : 0;  // the kept key sum is current
    }
  }
}
