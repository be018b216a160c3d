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
};

template <int T, int U>
__device__ __forceinline__ bool unit_front(const FusedParams &p,
                                           unsigned char *stage, int idx,
                                           int w, int lane,
                                           UnitFront<(T + U - 1) / U> &f) {
  constexpr int TW = (T + U - 1) / U;  // tiles per warp (at most)
  constexpr int R = 16 * T;
  const StageLayout L(R);
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
  //    two accumulator chains.
  float (&acc)[TW][4] = f.pr;
#pragma unroll
  for (int j = 0; j < TW; ++j) {
    float a2[4] = {0.f, 0.f, 0.f, 0.f};
    acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;
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
      }
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[j][e] += a2[e];
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
template <int T, int U>
__device__ __forceinline__ void unit_publish(unsigned char *garea,
                                             const UnitFront<(T + U - 1) / U> &f,
                                             int w, int lane) {
  if constexpr (U > 1) {
    const GroupLayout GL(U);
    float4 *XS4 = reinterpret_cast<float4 *>(garea + GL.xs);
    float4 *OX = reinterpret_cast<float4 *>(garea + GL.ox);
    if (lane < 4) XS4[w * 5 + lane] = make_float4(f.ref0, f.ref1, f.z0, f.z1);
#pragma unroll
    for (int mt = 0; mt < 8; ++mt)
      OX[(w * 8 + mt) * 32 + lane] =
          make_float4(f.o[mt][0], f.o[mt][1], f.o[mt][2], f.o[mt][3]);
  }
}

template <int T, int U, bool kOutBf16>
__device__ __forceinline__ void unit_back(const FusedParams &p,
                                          unsigned char *garea,
                                          UnitFront<(T + U - 1) / U> &f,
                                          int w, int lane, int bar_id) {
  constexpr int TW = (T + U - 1) / U;
  const GroupLayout GL(U);
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
      r[v] = XS4[v * 5 + (lane & 3)];
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
#pragma unroll
  for (int j = 0; j < TW; ++j) {
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
          const int pr = f.ps[j][hsel];
          if (pr <= wlo) {
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
      XW[w * 5 + 4] = make_uint4((uint32_t)best, (uint32_t)(best >> 32),
                                 (uint32_t)bi, 0u);
    group_bar(bar_id, 32 * U);
#pragma unroll
    for (int v = 0; v < U; ++v) {
      const uint4 a = XW[v * 5 + 4];
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
    }
  }
}
