// kvr_api.cu -- the C ABI of libkvr (include/kvr.h): argument validation,
// the host mirror of every live length, carving of the caller's device
// buffer, and kernel dispatch.  No device memory is allocated here.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <map>
#include <mutex>
#include <utility>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>
#include <array>
#include <vector>

#include "../../include/kvr.h"
#include "kvr_internal.h"

using kvr::CacheView;
using kvr::StepArgs;

namespace {

thread_local std::string g_err;

kvr_status fail(kvr_status st, const char *fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_err = buf;
  return st;
}

kvr_status cuda_fail(const char *where, cudaError_t e) {
  return fail(KVR_ECUDA, "%s: %s", where, cudaGetErrorString(e));
}

constexpr size_t kAlign = 256;
size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

int esize(kvr_dtype t) { return t == KVR_BF16 ? 2 : 4; }

bool desc_ok(const kvr_cache_desc *d) {
  if (!d) return false;
  if (d->n_seq < 1 || d->n_layers < 1 || d->n_kv_heads < 1) return false;
  if (d->group < 1 || d->group > 8) return false;
  if (d->head_dim != 64 && d->head_dim != 128) return false;
  if (d->capacity < 1 || d->capacity > (1 << 24)) return false;
  if (d->kv_dtype != KVR_BF16 && d->kv_dtype != KVR_F32) return false;
  if (d->out_dtype != KVR_BF16 && d->out_dtype != KVR_F32) return false;
  if (!(d->softmax_scale >= 0.f) || !std::isfinite(d->softmax_scale))
    return false;
  return true;
}

// Byte offsets of every array inside the cache buffer.
struct Layout {
  size_t K, V, score, pos, state, err, logits, rsum, total;
};

Layout layout_of(const kvr_cache_desc *d) {
  const size_t units = (size_t)d->n_seq * d->n_layers * d->n_kv_heads;
  const size_t rows = units * (size_t)d->capacity;
  const size_t srows = units * (size_t)kvr::round_up16(d->capacity);
  Layout l{};
  size_t off = 0;
  l.K = off;
  off = align_up(off + rows * d->head_dim * esize(d->kv_dtype));
  l.V = off;
  off = align_up(off + rows * d->head_dim * esize(d->kv_dtype));
  l.score = off;
  off = align_up(off + srows * sizeof(float));
  l.pos = off;
  off = align_up(off + srows * sizeof(int32_t));
  l.state = off;
  off = align_up(off + units * 4 * sizeof(int32_t));
  l.err = off;
  off = align_up(off + 16);
  l.logits = off;
  off = align_up(off + rows * d->group * sizeof(float));
  l.rsum = off;
  off = align_up(off + units * (size_t)d->head_dim * sizeof(float));
  l.total = off;
  return l;
}

}  // namespace

struct kvr_cache {
  kvr_cache_desc desc;
  CacheView view;
  std::vector<int32_t> len;       // host mirror [S][L]
  std::vector<int32_t> next_pos;  // host mirror [S][L]
  size_t bytes;
  uint64_t launches = 0;          // kernels launched through this handle
  bool fused = true;              // use the fused kernel where it applies
  int fused_groups = 0;           // units computed at once per SM (0: auto)
  int fused_group_warps = 0;      // warps per unit (0: auto)
  int chunk_groups = 0;           // chunked kernel: groups (0 auto, -1 off)
  int chunk_stages = 0;           // chunked kernel: stages per group (0 auto)
  int absorb_kernel = 0;          // 0 tcgen05, 1 mma.sync (kvr_absorb_chunk)
  int last_absorb = -1;           // kernel of the last kvr_absorb_chunk (0, 1, 2)
  int forks = 0;                  // live forks: the cache is read-only meanwhile
  int sm_count = 0;               // of the device, queried on first use
  int smem_optin = 0;
  std::map<int, std::pair<CUtensorMap, CUtensorMap>> tmaps;  // by box rows
  cudaEvent_t host_step_done = nullptr;  // last kvr_decode_step_host step
  bool host_step_recorded = false;
};

namespace {

// cuTensorMapEncodeTiled through the runtime's driver entry point (the
// library links no driver stub, so it also loads on hosts without a GPU).
PFN_cuTensorMapEncodeTiled_v12000 encode_tiled() {
  static std::once_flag once;
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  std::call_once(once, [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                         cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// 2-D view of a K or V slab: [units * cap rows][128 bf16], boxes of
// 64 columns x R rows, 128-byte swizzle (conflict-free ldmatrix).
bool encode_slab(CUtensorMap *m, void *base, size_t rows, int R) {
  auto fn = encode_tiled();
  if (!fn) return false;
  cuuint64_t dims[2] = {128, (cuuint64_t)rows};
  cuuint64_t strides[1] = {256};
  cuuint32_t box[2] = {64, (cuuint32_t)R};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The N candidates' tails as one 3-D tensor {128 elements, units * tcap rows,
// N candidates}: a box {64, T, Z} fetches T rows of Z candidates at once
// (Z = N unless given).
bool encode_tails3(CUtensorMap *m, void *base, size_t rows_per_cand, int n_cand,
                   int T, int Z = 0) {
  auto fn = encode_tiled();
  if (!fn) return false;
  cuuint64_t dims[3] = {128, (cuuint64_t)rows_per_cand, (cuuint64_t)n_cand};
  cuuint64_t strides[2] = {256, (cuuint64_t)rows_per_cand * 256};
  cuuint32_t box[3] = {64, (cuuint32_t)T, (cuuint32_t)(Z ? Z : n_cand)};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, base, dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The N candidates' tails as a 4-D tensor {128 elements, nt rows, units, N}
// (a unit's tail is tcap rows apart, a candidate's units * tcap): a box
// {64, round_up16(nt), 1, min(N, 2)} fetches the first nt rows of one unit's
// tails for two candidates and fills the rest of the box with zeros.
bool encode_tails4(CUtensorMap *m, void *base, int nt, int tcap, size_t units,
                   int n_cand) {
  auto fn = encode_tiled();
  if (!fn || nt < 1) return false;
  cuuint64_t dims[4] = {128, (cuuint64_t)nt, (cuuint64_t)units, (cuuint64_t)n_cand};
  cuuint64_t strides[3] = {256, (cuuint64_t)tcap * 256, (cuuint64_t)units * tcap * 256};
  cuuint32_t box[4] = {64, (cuuint32_t)kvr::round_up16(nt), 1,
                       (cuuint32_t)std::min(n_cand, 2)};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, base, dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The chunk's queries as a 4-D tensor {128 elements, G heads, H KV heads,
// tokens}: a box {64, G, 1, 128 / G} fetches the whole tokens that fill at
// most 128 rows (token * G + g) of one KV head.
bool encode_q4(CUtensorMap *m, const void *base, int G, int H, size_t tokens) {
  auto fn = encode_tiled();
  if (!fn || G < 1 || G > 8) return false;
  cuuint64_t dims[4] = {128, (cuuint64_t)G, (cuuint64_t)H, (cuuint64_t)tokens};
  cuuint64_t strides[3] = {256, (cuuint64_t)G * 256, (cuuint64_t)H * G * 256};
  cuuint32_t box[4] = {64, (cuuint32_t)G, 1, (cuuint32_t)(128 / G)};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base), dims, strides,
            box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

namespace {

cudaStream_t as_stream(void *s) { return reinterpret_cast<cudaStream_t>(s); }

kvr_status check_layers(const kvr_cache *c, int lb, int le) {
  if (lb < 0 || le > c->desc.n_layers || lb >= le)
    return fail(KVR_EINVAL, "layer range [%d, %d) outside [0, %d)", lb, le,
                c->desc.n_layers);
  return KVR_OK;
}

// Largest live length over (all sequences) x (layers [lb, le)).
int max_len(const kvr_cache *c, int lb, int le) {
  int m = 0;
  for (int s = 0; s < c->desc.n_seq; ++s)
    for (int l = lb; l < le; ++l)
      m = std::max(m, c->len[(size_t)s * c->desc.n_layers + l]);
  return m;
}

kvr_status check_step(kvr_cache *c, int lb, int le, const void *q,
                      const void *k_new, const void *v_new, void *out) {
  if (!c) return fail(KVR_EINVAL, "null cache");
  if (c->forks) return fail(KVR_ESTATE, "the cache has a live fork");
  kvr_status st = check_layers(c, lb, le);
  if (st != KVR_OK) return st;
  if (!q || !k_new || !v_new || !out)
    return fail(KVR_EINVAL, "null q, k_new, v_new or out");
  const int m = max_len(c, lb, le);
  if (m + 1 > c->desc.capacity)
    return fail(KVR_ECAPACITY, "a unit holds %d rows; capacity %d is full", m,
                c->desc.capacity);
  for (int s = 0; s < c->desc.n_seq; ++s)
    for (int l = lb; l < le; ++l)
      if (c->next_pos[(size_t)s * c->desc.n_layers + l] == INT32_MAX)
        return fail(KVR_ECAPACITY, "position counter exhausted");
  return KVR_OK;
}

kvr_status check_evict(int budget, int window) {
  if (budget < 0 || window < 0 || (long long)budget + window < 1 ||
      (long long)budget + window > (1 << 24))
    return fail(KVR_EINVAL, "bad budget %d / window %d", budget, window);
  return KVR_OK;
}

void mirror_append(kvr_cache *c, int lb, int le) {
  for (int s = 0; s < c->desc.n_seq; ++s)
    for (int l = lb; l < le; ++l) {
      const size_t i = (size_t)s * c->desc.n_layers + l;
      c->len[i] += 1;
      c->next_pos[i] += 1;
    }
}

void mirror_evict(kvr_cache *c, int lb, int le, int budget, int window) {
  for (int s = 0; s < c->desc.n_seq; ++s)
    for (int l = lb; l < le; ++l) {
      int32_t &n = c->len[(size_t)s * c->desc.n_layers + l];
      n = std::min<long long>(n, (long long)budget + window);
    }
}

StepArgs step_args(const kvr_cache *c, int lb, int le, const void *q,
                   const void *k_new, const void *v_new, void *out) {
  StepArgs a{};
  a.lb = lb;
  a.nl = le - lb;
  a.q = q;
  a.k_new = k_new;
  a.v_new = v_new;
  a.out = out;
  a.max_rows = max_len(c, lb, le) + 1;
  return a;
}

}  // namespace

namespace {

bool aligned16(const void *p) {
  return reinterpret_cast<uintptr_t>(p) % 16 == 0;
}

// Launch the fused kernel if this call qualifies; returns false (and does
// nothing) if it does not, true with *err set otherwise.
// Device facts the dispatch needs, queried once per handle.
bool device_facts(kvr_cache *c) {
  if (c->sm_count) return true;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&c->sm_count, cudaDevAttrMultiProcessorCount,
                             dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&c->smem_optin,
                             cudaDevAttrMaxSharedMemoryPerBlockOptin,
                             dev) != cudaSuccess) {
    c->sm_count = 0;
    return false;
  }
  return true;
}

// The K and V tensor maps with boxes of `box_rows` rows (created on first
// use and kept in the handle); NULL if they cannot be encoded.
const std::pair<CUtensorMap, CUtensorMap> *slab_maps(kvr_cache *c,
                                                      int box_rows) {
  auto it = c->tmaps.find(box_rows);
  if (it == c->tmaps.end()) {
    const CacheView &v = c->view;
    const size_t rows = (size_t)v.S * v.L * v.H * v.cap;
    std::pair<CUtensorMap, CUtensorMap> maps;
    if (!encode_slab(&maps.first, v.K, rows, box_rows) ||
        !encode_slab(&maps.second, v.V, rows, box_rows))
      return nullptr;
    it = c->tmaps.emplace(box_rows, maps).first;
  }
  return &it->second;
}

bool try_fused(kvr_cache *c, const StepArgs &a, bool evict, int budget,
               int window, cudaStream_t stream, cudaError_t *err,
               bool rkv = false, float lam = 0.f) {
  const CacheView &v = c->view;
  if (!c->fused || !v.kv_bf16 || v.d != 128 || v.G > 8) return false;
  if (a.max_rows > kvr::fused_max_rows()) return false;
  if (evict && (long long)a.max_rows > (long long)budget + window + 1)
    return false;
  const size_t rows = (size_t)v.S * v.L * v.H * v.cap;
  if (rows >= (size_t)INT32_MAX) return false;
  if (!aligned16(a.q) || !aligned16(a.k_new) || !aligned16(a.v_new) ||
      !aligned16(a.out))
    return false;
  if (!device_facts(c)) return false;
  const int R = kvr::round_up16(a.max_rows);
  const int Rb = std::max(8, (a.max_rows - 1 + 7) / 8 * 8);
  const int U = kvr::fused_group_warps(R, c->fused_group_warps);
  if (U < 1) return false;
  const int stage = kvr::fused_stage_bytes(R, rkv);
  const int gbytes = kvr::fused_group_bytes(U, rkv);
  const int avail = c->smem_optin - 1024 /*alignment*/ - 512 /*static*/;
  // Consumer groups hold a stage only while reading it; the rest of shared
  // memory is ring.  By default as many groups as there are stages (at most
  // four; measured best), a tuned count as long as two stages remain.
  const int max_groups = std::min(kvr::fused_max_groups(),
                                  (kvr::fused_max_threads() / 32 -
                                   kvr::fused_producer_warps()) / U);
  const bool tuned = c->fused_groups > 0;
  int n_groups = std::min(max_groups, tuned ? c->fused_groups : 4);
  int n_stages = 0;
  for (; n_groups >= 1; --n_groups) {
    n_stages = std::min(8, (avail - n_groups * gbytes) / stage);
    if (n_stages >= (tuned ? 2 : std::max(2, n_groups))) break;
  }
  if (n_groups < 1 || n_stages < 2) return false;
  const std::pair<CUtensorMap, CUtensorMap> *maps = slab_maps(c, Rb);
  if (!maps) return false;
  kvr::FusedParams p{};
  p.c = v;
  p.q = static_cast<const __nv_bfloat16 *>(a.q);
  p.k_new = static_cast<const __nv_bfloat16 *>(a.k_new);
  p.v_new = static_cast<const __nv_bfloat16 *>(a.v_new);
  p.out = a.out;
  p.lb = a.lb;
  p.nl = a.nl;
  p.R = R;
  p.Rb = Rb;
  p.n_stages = n_stages;
  p.n_groups = n_groups;
  p.group_warps = U;
  p.budget = budget;
  p.window = window;
  p.evict = evict ? 1 : 0;
  p.scale_log2e = v.scale * 1.4426950408889634f;
  p.inv_g = 1.f / (float)v.G;
  p.rkv = rkv ? 1 : 0;
  p.lam = lam;
  const int units = v.S * a.nl * v.H;
  const int grid = std::min(c->sm_count, units);
  *err = kvr::launch_fused_step(maps->first, maps->second, p, grid,
                                n_stages * stage + n_groups * gbytes + 1024,
                                stream);
  return true;
}

// Launch the streaming fused step (longer units) if this call qualifies.
bool try_stream(kvr_cache *c, const StepArgs &a, bool evict, int budget,
                int window, cudaStream_t stream, cudaError_t *err) {
  const CacheView &v = c->view;
  if (!c->fused || !v.kv_bf16 || v.d != 128 || v.G > 8) return false;
  if (a.max_rows > kvr::stream_max_rows()) return false;
  if (evict && (long long)a.max_rows > (long long)budget + window + 1)
    return false;
  const size_t rows = (size_t)v.S * v.L * v.H * v.cap;
  if (rows >= (size_t)INT32_MAX) return false;
  if (!aligned16(a.q) || !aligned16(a.k_new) || !aligned16(a.v_new) ||
      !aligned16(a.out))
    return false;
  if (!device_facts(c)) return false;
  if (kvr::stream_smem_bytes(a.max_rows) + 512 > (size_t)c->smem_optin)
    return false;
  const std::pair<CUtensorMap, CUtensorMap> *maps =
      slab_maps(c, kvr::stream_box_rows());
  if (!maps) return false;
  kvr::StreamParams p{};
  p.c = v;
  p.q = static_cast<const __nv_bfloat16 *>(a.q);
  p.k_new = static_cast<const __nv_bfloat16 *>(a.k_new);
  p.v_new = static_cast<const __nv_bfloat16 *>(a.v_new);
  p.out = a.out;
  p.lb = a.lb;
  p.nl = a.nl;
  p.n_max = a.max_rows;
  p.budget = budget;
  p.window = window;
  p.evict = evict ? 1 : 0;
  p.scale_log2e = v.scale * 1.4426950408889634f;
  *err = kvr::launch_stream_step(maps->first, maps->second, p, stream);
  return true;
}

// Consumer groups and ring stages per group of the chunked kernel for jobs
// of up to n_max rows: the first of (4,2) (3,3) (3,2) (2,3) (2,2) (1,3)
// (1,2) that fits in shared memory (more groups first: measured), or the
// tuned choice.
bool chunk_config(const kvr_cache *c, int n_max, int *groups, int *stages) {
  static const int order[7][2] = {{4, 2}, {3, 3}, {3, 2}, {2, 3},
                                  {2, 2}, {1, 3}, {1, 2}};
  const size_t limit = (size_t)c->smem_optin - 512;
  const int tg = c->chunk_groups, ts = c->chunk_stages;
  for (const auto &o : order) {
    const int g = tg > 0 ? tg : o[0], s = ts > 0 ? ts : o[1];
    if (g > kvr::chunk_max_groups() || s > kvr::chunk_max_stages()) continue;
    if (kvr::chunk_smem_bytes(n_max, g, s) <= limit) {
      *groups = g;
      *stages = s;
      return true;
    }
  }
  return false;
}

// Launch the chunked step for plain units if this call qualifies.
bool try_chunked(kvr_cache *c, const StepArgs &a, bool evict, int budget,
                 int window, cudaStream_t stream, cudaError_t *err) {
  const CacheView &v = c->view;
  if (!c->fused || c->chunk_groups < 0 || !v.kv_bf16 || v.d != 128 ||
      v.G > 8)
    return false;
  if (a.max_rows > kvr::chunk_max_rows()) return false;
  if (evict && (long long)a.max_rows > (long long)budget + window + 1)
    return false;
  const size_t rows = (size_t)v.S * v.L * v.H * v.cap;
  if (rows >= (size_t)INT32_MAX) return false;
  if (!aligned16(a.q) || !aligned16(a.k_new) || !aligned16(a.v_new) ||
      !aligned16(a.out))
    return false;
  if (!device_facts(c)) return false;
  kvr::ChunkParams p{};
  if (!chunk_config(c, a.max_rows, &p.n_groups, &p.n_stages)) return false;
  const std::pair<CUtensorMap, CUtensorMap> *maps =
      slab_maps(c, kvr::chunk_box_rows());
  if (!maps) return false;
  p.c = v;
  p.fork = 0;
  p.q = static_cast<const __nv_bfloat16 *>(a.q);
  p.k_new = static_cast<const __nv_bfloat16 *>(a.k_new);
  p.v_new = static_cast<const __nv_bfloat16 *>(a.v_new);
  p.out = a.out;
  p.lb = a.lb;
  p.nl = a.nl;
  p.n_jobs = v.S * a.nl * v.H;
  p.n_max = a.max_rows;
  p.budget = budget;
  p.window = window;
  p.evict = evict ? 1 : 0;
  p.scale_log2e = v.scale * 1.4426950408889634f;
  p.inv_g = 1.f / (float)v.G;
  const int grid = std::min(c->sm_count, p.n_jobs);
  *err = kvr::launch_chunk_step(maps->first, maps->second, nullptr, nullptr, p,
                                grid, stream);
  return true;
}

// Splits for kvr_decode_attend: about two waves of the partial kernel (three
// CTAs per SM), never less than 256 rows per split.
int auto_splits(const kvr_cache *c, int lb, int le) {
  const int units = c->desc.n_seq * (le - lb) * c->desc.n_kv_heads;
  const int rows = max_len(c, lb, le) + 1;
  const int sms = c->sm_count > 0 ? c->sm_count : 148;
  const int want = (2 * 3 * sms + units - 1) / units;
  return std::max(1, std::min(want, (rows + 255) / 256));
}

}  // namespace

extern "C" {

size_t kvr_decode_attend_workspace_bytes(const kvr_cache *c, int lb, int le,
                                         int n_splits) {
  if (!c || lb < 0 || le > c->desc.n_layers || lb >= le || n_splits < 0)
    return 0;
  if (n_splits == 0) {
    device_facts(const_cast<kvr_cache *>(c));
    n_splits = auto_splits(c, lb, le);
  }
  return kvr::split_workspace_bytes(c->view, le - lb, n_splits);
}

kvr_status kvr_decode_attend(kvr_cache *c, int lb, int le, const void *q,
                             const void *k_new, const void *v_new, void *out,
                             int n_splits, void *workspace,
                             size_t workspace_bytes, void *stream) {
  kvr_status st = check_step(c, lb, le, q, k_new, v_new, out);
  if (st != KVR_OK) return st;
  const CacheView &v = c->view;
  if (!v.kv_bf16 || v.d != 128 || v.G > 8)
    return fail(KVR_EINVAL, "kvr_decode_attend needs bf16, head_dim 128, G<=8");
  if (n_splits < 0 || n_splits > 4096)
    return fail(KVR_EINVAL, "bad n_splits %d", n_splits);
  if (!aligned16(q) || !aligned16(k_new) || !aligned16(v_new) ||
      !aligned16(out) || !aligned16(workspace))
    return fail(KVR_EINVAL, "q, k_new, v_new, out and workspace must be "
                "16-byte aligned");
  const size_t rows = (size_t)v.S * v.L * v.H * v.cap;
  if (rows >= (size_t)INT32_MAX)
    return fail(KVR_EINVAL, "slab of %zu rows is beyond the TMA coordinate "
                "range", rows);
  if (!device_facts(c)) return fail(KVR_ECUDA, "cannot query the device");
  if (n_splits == 0) n_splits = auto_splits(c, lb, le);
  const size_t need = kvr::split_workspace_bytes(v, le - lb, n_splits);
  if (!workspace || workspace_bytes < need)
    return fail(KVR_ENOMEM, "workspace of %zu bytes < required %zu",
                workspace_bytes, need);
  const int box = kvr::split_rows_per_stage();
  const std::pair<CUtensorMap, CUtensorMap> *maps = slab_maps(c, box);
  if (!maps) return fail(KVR_ECUDA, "cannot encode the TMA descriptors");
  kvr::SplitParams p{};
  p.c = v;
  p.q = static_cast<const __nv_bfloat16 *>(q);
  p.k_new = static_cast<const __nv_bfloat16 *>(k_new);
  p.v_new = static_cast<const __nv_bfloat16 *>(v_new);
  p.lb = lb;
  p.nl = le - lb;
  p.n_splits = n_splits;
  p.ws = static_cast<float *>(workspace);
  p.scale_log2e = v.scale * 1.4426950408889634f;
  cudaError_t e = kvr::launch_split_attend(maps->first, maps->second, p, out,
                                           as_stream(stream));
  if (e != cudaSuccess) return cuda_fail("kvr_decode_attend", e);
  c->launches += 2;
  mirror_append(c, lb, le);
  return KVR_OK;
}

size_t kvr_cache_required_bytes(const kvr_cache_desc *desc) {
  if (!desc_ok(desc)) return 0;
  return layout_of(desc).total;
}

kvr_status kvr_cache_create(const kvr_cache_desc *desc, void *dev_buf,
                            size_t bytes, void *stream, kvr_cache **out) {
  if (!out) return fail(KVR_EINVAL, "null output handle");
  *out = nullptr;
  if (!desc_ok(desc)) return fail(KVR_EINVAL, "invalid cache descriptor");
  if (!dev_buf) return fail(KVR_EINVAL, "null device buffer");
  if (reinterpret_cast<uintptr_t>(dev_buf) % kAlign)
    return fail(KVR_EINVAL, "device buffer not %zu-byte aligned", kAlign);
  const Layout lay = layout_of(desc);
  if (bytes < lay.total)
    return fail(KVR_ENOMEM, "buffer of %zu bytes < required %zu", bytes,
                lay.total);
  kvr_cache *c = new (std::nothrow) kvr_cache();
  if (!c) return fail(KVR_ENOMEM, "host allocation failed");
  c->desc = *desc;
  c->bytes = bytes;
  char *b = static_cast<char *>(dev_buf);
  CacheView &v = c->view;
  v.K = b + lay.K;
  v.V = b + lay.V;
  v.score = reinterpret_cast<float *>(b + lay.score);
  v.pos = reinterpret_cast<int32_t *>(b + lay.pos);
  v.state = reinterpret_cast<int32_t *>(b + lay.state);
  v.err = reinterpret_cast<unsigned *>(b + lay.err);
  v.logits = reinterpret_cast<float *>(b + lay.logits);
  v.rsum = reinterpret_cast<float *>(b + lay.rsum);
  v.S = desc->n_seq;
  v.L = desc->n_layers;
  v.H = desc->n_kv_heads;
  v.G = desc->group;
  v.d = desc->head_dim;
  v.cap = desc->capacity;
  v.sstride = kvr::round_up16(desc->capacity);
  v.scale = desc->softmax_scale > 0.f
                ? desc->softmax_scale
                : (float)(1.0 / std::sqrt((double)desc->head_dim));
  v.kv_bf16 = desc->kv_dtype == KVR_BF16;
  v.out_bf16 = desc->out_dtype == KVR_BF16;
  v.wait_ns = kvr::kDefaultWaitNs;
  v.hold_first = 0;
  c->len.assign((size_t)v.S * v.L, 0);
  c->next_pos.assign((size_t)v.S * v.L, 0);
  cudaError_t e = kvr::launch_init(v, as_stream(stream));
  if (e != cudaSuccess) {
    delete c;
    return cuda_fail("kvr_cache_create", e);
  }
  *out = c;
  return KVR_OK;
}

void kvr_cache_destroy(kvr_cache *cache) {
  if (cache && cache->host_step_done) cudaEventDestroy(cache->host_step_done);
  delete cache;
}

kvr_status kvr_cache_load(kvr_cache *c, int seq, const void *k, const void *v,
                          int n_rows, int first_pos, void *stream) {
  if (!c) return fail(KVR_EINVAL, "null cache");
  if (c->forks) return fail(KVR_ESTATE, "the cache has a live fork");
  if (seq < 0 || seq >= c->desc.n_seq)
    return fail(KVR_EINVAL, "sequence %d outside [0, %d)", seq, c->desc.n_seq);
  if (n_rows < 0 || first_pos < 0 ||
      (long long)first_pos + n_rows >= INT32_MAX)
    return fail(KVR_EINVAL, "bad prompt length %d / first position %d", n_rows,
                first_pos);
  if (n_rows > c->desc.capacity)
    return fail(KVR_ECAPACITY, "prompt of %d rows > capacity %d", n_rows,
                c->desc.capacity);
  if (n_rows > 0 && (!k || !v)) return fail(KVR_EINVAL, "null k or v");
  if ((reinterpret_cast<uintptr_t>(k) | reinterpret_cast<uintptr_t>(v)) % 16)
    return fail(KVR_EINVAL, "k and v must be 16-byte aligned");
  cudaError_t e =
      kvr::launch_load(c->view, seq, k, v, n_rows, first_pos, as_stream(stream));
  if (e != cudaSuccess) return cuda_fail("kvr_cache_load", e);
  c->launches += 1;
  for (int l = 0; l < c->desc.n_layers; ++l) {
    c->len[(size_t)seq * c->desc.n_layers + l] = n_rows;
    c->next_pos[(size_t)seq * c->desc.n_layers + l] = first_pos + n_rows;
  }
  return KVR_OK;
}

kvr_status kvr_decode_attend_score(kvr_cache *c, int lb, int le, const void *q,
                                   const void *k_new, const void *v_new,
                                   void *out, void *stream) {
  kvr_status st = check_step(c, lb, le, q, k_new, v_new, out);
  if (st != KVR_OK) return st;
  StepArgs a = step_args(c, lb, le, q, k_new, v_new, out);
  cudaError_t e = cudaSuccess;
  if (!try_fused(c, a, false, 0, 0, as_stream(stream), &e) &&
      !try_chunked(c, a, false, 0, 0, as_stream(stream), &e) &&
      !try_stream(c, a, false, 0, 0, as_stream(stream), &e))
    e = kvr::launch_attend_score_generic(c->view, a, as_stream(stream));
  if (e != cudaSuccess) return cuda_fail("kvr_decode_attend_score", e);
  c->launches += 1;
  mirror_append(c, lb, le);
  return KVR_OK;
}

kvr_status kvr_cache_copy_sequences(kvr_cache *dst, const int32_t *dst_seqs,
                                    const kvr_cache *src,
                                    const int32_t *src_seqs, int n,
                                    void *stream) {
  if (!dst || !src) return fail(KVR_EINVAL, "null cache");
  if (n < 0) return fail(KVR_EINVAL, "negative count %d", n);
  if (n == 0) return KVR_OK;
  if (!dst_seqs || !src_seqs) return fail(KVR_EINVAL, "null sequence list");
  if (dst->forks || src->forks) return fail(KVR_ESTATE, "a cache has a live fork");
  const kvr_cache_desc &a = src->desc, &b = dst->desc;
  if (a.n_layers != b.n_layers || a.n_kv_heads != b.n_kv_heads ||
      a.head_dim != b.head_dim || a.kv_dtype != b.kv_dtype)
    return fail(KVR_EINVAL, "the caches' layers, KV heads, head_dim or "
                "kv_dtype differ");
  const int L = a.n_layers;
  std::vector<char> taken(b.n_seq, 0), read(a.n_seq, 0);
  for (int i = 0; i < n; ++i) {
    const int s = src_seqs[i], d = dst_seqs[i];
    if (s < 0 || s >= a.n_seq || d < 0 || d >= b.n_seq)
      return fail(KVR_EINVAL, "pair %d (%d -> %d) outside the caches", i, s, d);
    if (taken[d]) return fail(KVR_EINVAL, "sequence %d is written twice", d);
    taken[d] = 1;
    read[s] = 1;
    for (int l = 0; l < L; ++l)
      if (src->len[(size_t)s * L + l] > b.capacity)
        return fail(KVR_ECAPACITY, "sequence %d holds %d rows > capacity %d",
                    s, src->len[(size_t)s * L + l], b.capacity);
  }
  if (dst == src)
    for (int i = 0; i < n; ++i)
      if (read[dst_seqs[i]])
        return fail(KVR_EINVAL, "sequence %d is both read and written",
                    dst_seqs[i]);
  const int row_bytes = a.head_dim * esize(a.kv_dtype);
  kvr::SeqPairs pairs;
  for (int i0 = 0; i0 < n; i0 += kvr::kMaxSeqPairs) {
    const int m = std::min(kvr::kMaxSeqPairs, n - i0);
    for (int i = 0; i < m; ++i) {
      pairs.src[i] = src_seqs[i0 + i];
      pairs.dst[i] = dst_seqs[i0 + i];
    }
    cudaError_t e = kvr::launch_copy_seqs(dst->view, src->view, pairs, m,
                                          row_bytes, as_stream(stream));
    if (e != cudaSuccess) return cuda_fail("kvr_cache_copy_sequences", e);
    dst->launches += 1;
  }
  for (int i = 0; i < n; ++i)
    for (int l = 0; l < L; ++l) {
      dst->len[(size_t)dst_seqs[i] * L + l] = src->len[(size_t)src_seqs[i] * L + l];
      dst->next_pos[(size_t)dst_seqs[i] * L + l] =
          src->next_pos[(size_t)src_seqs[i] * L + l];
    }
  return KVR_OK;
}

kvr_status kvr_cache_set_absorb_kernel(kvr_cache *c, int kernel) {
  if (!c) return fail(KVR_EINVAL, "null cache");
  if (kernel < 0 || kernel > 1) return fail(KVR_EINVAL, "kernel must be 0 or 1");
  c->absorb_kernel = kernel;
  return KVR_OK;
}

kvr_status kvr_cache_set_wait_limit(kvr_cache *c, uint64_t ns) {
  if (!c) return fail(KVR_EINVAL, "null cache");
  if (ns > kvr::kDefaultWaitNs)
    return fail(KVR_EINVAL, "wait limit %llu ns above the %llu ns default",
                (unsigned long long)ns, kvr::kDefaultWaitNs);
  c->view.wait_ns = ns ? ns : kvr::kDefaultWaitNs;
  return KVR_OK;
}

kvr_status kvr_cache_set_hold_first_unit(kvr_cache *c, int enable) {
  if (!c) return fail(KVR_EINVAL, "null cache");
  c->view.hold_first = enable != 0;
  return KVR_OK;
}

kvr_status kvr_cache_set_fused(kvr_cache *c, int enable) {
  if (!c) return fail(KVR_EINVAL, "null cache");
  c->fused = enable != 0;
  return KVR_OK;
}

kvr_status kvr_cache_set_fused_tuning(kvr_cache *c, int groups,
                                      int group_warps) {
  if (!c) return fail(KVR_EINVAL, "null cache");
  if (groups < 0 || groups > 4 || group_warps < 0 || group_warps > 8)
    return fail(KVR_EINVAL, "tuning (%d, %d) outside [0, 4] x [0, 8]", groups,
                group_warps);
  c->fused_groups = groups;
  c->fused_group_warps = group_warps;
  return KVR_OK;
}

kvr_status kvr_cache_set_chunk_tuning(kvr_cache *c, int groups, int stages) {
  if (!c) return fail(KVR_EINVAL, "null cache");
  if (groups < -1 || groups > 4 || stages < 0 || stages > 4 || stages == 1)
    return fail(KVR_EINVAL, "chunk tuning (%d, %d) outside [-1, 4] x "
                "{0, 2, 3, 4}", groups, stages);
  c->chunk_groups = groups;
  c->chunk_stages = stages;
  return KVR_OK;
}

}  // extern "C"

int kvr::report_cuda_error(const char *where, cudaError_t e) {
  return cuda_fail(where, e);
}

int kvr::report_error(int st, const char *msg) {
  return fail(static_cast<kvr_status>(st), "%s", msg);
}

int kvr::decode_attend_score_ext(kvr_cache *c, int lb, int le, const void *q,
                                 const void *k_new, const void *v_new,
                                 void *out, float *ext, size_t ext_floats,
                                 void *stream) {
  kvr_status st = check_step(c, lb, le, q, k_new, v_new, out);
  if (st != KVR_OK) return st;
  if (!ext) return fail(KVR_EINVAL, "null scratch");
  StepArgs a = step_args(c, lb, le, q, k_new, v_new, out);
  const size_t need =
      (size_t)c->desc.n_seq * a.nl * c->desc.n_kv_heads * c->desc.group *
      (size_t)a.max_rows;
  if (need > ext_floats)
    return fail(KVR_EINVAL,
                "this call needs %zu bytes of logit scratch (%d seq x %d layers"
                " x %d heads x G=%d x %d rows x 4 B); the static scratch holds "
                "%zu bytes",
                need * sizeof(float), c->desc.n_seq, a.nl,
                c->desc.n_kv_heads, c->desc.group, a.max_rows,
                ext_floats * sizeof(float));
  cudaError_t e = kvr::launch_attend_score_ext_scratch(c->view, a, ext,
                                                       as_stream(stream));
  if (e != cudaSuccess) return cuda_fail("kvr_decode_attend_score_noalloc", e);
  c->launches += 1;
  mirror_append(c, lb, le);
  return KVR_OK;
}

extern "C" {

kvr_status kvr_evict_compact(kvr_cache *c, int lb, int le, int budget,
                             int window, void *stream) {
  if (!c) return fail(KVR_EINVAL, "null cache");
  if (c->forks) return fail(KVR_ESTATE, "the cache has a live fork");
  kvr_status st = check_layers(c, lb, le);
  if (st != KVR_OK) return st;
  st = check_evict(budget, window);
  if (st != KVR_OK) return st;
  const int m = max_len(c, lb, le);
  if (m <= budget + window) return KVR_OK;  // nothing exceeds B + W
  cudaError_t e = kvr::launch_evict_generic(c->view, lb, le - lb, m, budget,
                                            window, as_stream(stream));
  if (e != cudaSuccess) return cuda_fail("kvr_evict_compact", e);
  c->launches += 1;
  mirror_evict(c, lb, le, budget, window);
  return KVR_OK;
}

kvr_status kvr_evict_compact_rkv(kvr_cache *c, int lb, int le, int budget,
                                 int window, float lambda, void *stream) {
  if (!c) return fail(KVR_EINVAL, "null cache");
  if (c->forks) return fail(KVR_ESTATE, "the cache has a live fork");
  kvr_status st = check_layers(c, lb, le);
  if (st != KVR_OK) return st;
  st = check_evict(budget, window);
  if (st != KVR_OK) return st;
  if (!(lambda >= 0.f && lambda <= 1.f))
    return fail(KVR_EINVAL, "mix weight %g outside [0, 1]", (double)lambda);
  const int m = max_len(c, lb, le);
  if (m <= budget + window) return KVR_OK;
  cudaError_t e = kvr::launch_evict_rkv(c->view, lb, le - lb, m, budget,
                                        window, lambda, as_stream(stream));
  if (e != cudaSuccess) return cuda_fail("kvr_evict_compact_rkv", e);
  c->launches += 1;
  mirror_evict(c, lb, le, budget, window);
  return KVR_OK;
}

kvr_status kvr_absorb_chunk(kvr_cache *c, int lb, int le, int chunk,
                            const void *q, const void *k_new,
                            const void *v_new, void *out, int budget,
                            int window, int evict, void *stream) {
  if (!c) return fail(KVR_EINVAL, "null cache");
  if (c->forks) return fail(KVR_ESTATE, "the cache has a live fork");
  kvr_status st = check_layers(c, lb, le);
  if (st != KVR_OK) return st;
  if (!q || !k_new || !v_new || !out)
    return fail(KVR_EINVAL, "null q, k_new, v_new or out");
  if (chunk < 1) return fail(KVR_EINVAL, "chunk of %d tokens", chunk);
  if (evict) {
    st = check_evict(budget, window);
    if (st != KVR_OK) return st;
  }
  const int m = max_len(c, lb, le);
  if ((long long)m + chunk > c->desc.capacity)
    return fail(KVR_ECAPACITY, "a unit holds %d rows; %d more exceed capacity "
                "%d", m, chunk, c->desc.capacity);
  for (int s = 0; s < c->desc.n_seq; ++s)
    for (int l = lb; l < le; ++l)
      if ((long long)c->next_pos[(size_t)s * c->desc.n_layers + l] + chunk >=
          INT32_MAX)
        return fail(KVR_ECAPACITY, "position counter exhausted");
  const CacheView &v = c->view;
  if (c->fused && v.kv_bf16 && v.d == 128 && v.G <= 8 &&
      chunk <= kvr::absorb_max_chunk() && m + chunk <= kvr::absorb_max_rows() &&
      aligned16(q) && aligned16(k_new) && aligned16(v_new) && aligned16(out)) {
    kvr::AbsorbParams p{};
    p.c = v;
    p.q = static_cast<const __nv_bfloat16 *>(q);
    p.k_new = static_cast<const __nv_bfloat16 *>(k_new);
    p.v_new = static_cast<const __nv_bfloat16 *>(v_new);
    p.out = out;
    p.lb = lb;
    p.nl = le - lb;
    p.chunk = chunk;
    p.max_rows = m + chunk;
    p.budget = budget;
    p.window = window;
    p.evict = evict ? 1 : 0;
    p.scale_log2e = v.scale * 1.4426950408889634f;
    p.inv_g = 1.f / (float)v.G;
    CUtensorMap tmq;
    const bool have_q = encode_q4(&tmq, q, v.G, v.H, (size_t)v.S * p.nl * chunk);
    int ran = 1;
    cudaError_t e = kvr::launch_absorb(p, c->absorb_kernel, have_q ? &tmq : nullptr,
                                       as_stream(stream), &ran);
    if (e != cudaSuccess) return cuda_fail("kvr_absorb_chunk", e);
    c->last_absorb = ran;
    c->launches += 1;
    for (int j = 0; j < chunk; ++j) mirror_append(c, lb, le);
    if (evict) mirror_evict(c, lb, le, budget, window);
    return KVR_OK;
  }
  // Token by token: each launch appends token j of every unit and attends
  // over every live row, adding to the scores (eviction deferred).
  c->last_absorb = 2;
  for (int j = 0; j < chunk; ++j) {
    StepArgs a = step_args(c, lb, le, q, k_new, v_new, out);
    a.chunk = chunk;
    a.tok = j;
    cudaError_t e = kvr::launch_attend_score_generic(c->view, a, as_stream(stream));
    if (e != cudaSuccess) return cuda_fail("kvr_absorb_chunk", e);
    c->launches += 1;
    mirror_append(c, lb, le);
  }
  return evict ? kvr_evict_compact(c, lb, le, budget, window, stream) : KVR_OK;
}

kvr_status kvr_decode_step(kvr_cache *c, int lb, int le, const void *q,
                           const void *k_new, const void *v_new, void *out,
                           int budget, int window, void *stream) {
  kvr_status st = check_step(c, lb, le, q, k_new, v_new, out);
  if (st != KVR_OK) return st;
  st = check_evict(budget, window);
  if (st != KVR_OK) return st;
  StepArgs a = step_args(c, lb, le, q, k_new, v_new, out);
  cudaError_t e = cudaSuccess;
  if (try_fused(c, a, true, budget, window, as_stream(stream), &e) ||
      try_chunked(c, a, true, budget, window, as_stream(stream), &e) ||
      try_stream(c, a, true, budget, window, as_stream(stream), &e)) {
    if (e != cudaSuccess) return cuda_fail("kvr_decode_step", e);
    c->launches += 1;
    mirror_append(c, lb, le);
    mirror_evict(c, lb, le, budget, window);
    return KVR_OK;
  }
  st = kvr_decode_attend_score(c, lb, le, q, k_new, v_new, out, stream);
  if (st != KVR_OK) return st;
  return kvr_evict_compact(c, lb, le, budget, window, stream);
}

kvr_status kvr_decode_step_rkv(kvr_cache *c, int lb, int le, const void *q,
                               const void *k_new, const void *v_new,
                               void *out, int budget, int window, float lambda,
                               void *stream) {
  kvr_status st = check_step(c, lb, le, q, k_new, v_new, out);
  if (st != KVR_OK) return st;
  st = check_evict(budget, window);
  if (st != KVR_OK) return st;
  if (!(lambda >= 0.f && lambda <= 1.f))
    return fail(KVR_EINVAL, "mix weight %g outside [0, 1]", (double)lambda);
  StepArgs a = step_args(c, lb, le, q, k_new, v_new, out);
  cudaError_t e = cudaSuccess;
  if (try_fused(c, a, true, budget, window, as_stream(stream), &e, true,
                lambda)) {
    if (e != cudaSuccess) return cuda_fail("kvr_decode_step_rkv", e);
    c->launches += 1;
    mirror_append(c, lb, le);
    mirror_evict(c, lb, le, budget, window);
    return KVR_OK;
  }
  st = kvr_decode_attend_score(c, lb, le, q, k_new, v_new, out, stream);
  if (st != KVR_OK) return st;
  return kvr_evict_compact_rkv(c, lb, le, budget, window, lambda, stream);
}

kvr_status kvr_decode_step_host(kvr_cache *c, int lb, int le,
                                const void *q_host, const void *k_new_host,
                                const void *v_new_host, void *out_host,
                                void *q_dev, void *k_new_dev, void *v_new_dev,
                                void *out_dev, int budget, int window,
                                void *stream) {
  if (!q_host || !k_new_host || !v_new_host || !out_host)
    return fail(KVR_EINVAL, "null host q, k_new, v_new or out");
  kvr_status st = check_step(c, lb, le, q_dev, k_new_dev, v_new_dev, out_dev);
  if (st != KVR_OK) return st;
  st = check_evict(budget, window);
  if (st != KVR_OK) return st;
  const kvr_cache_desc &d = c->desc;
  const size_t rows = (size_t)d.n_seq * (le - lb) * d.n_kv_heads;
  const size_t row_kv = (size_t)d.head_dim * esize(d.kv_dtype);
  const size_t qb = rows * d.group * row_kv, kb = rows * row_kv;
  const size_t ob = rows * d.group * d.head_dim * esize(d.out_dtype);
  cudaStream_t s = as_stream(stream);
  cudaError_t e = cudaMemcpyAsync(q_dev, q_host, qb, cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(k_new_dev, k_new_host, kb, cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(v_new_dev, v_new_host, kb, cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess && !c->host_step_done)
    e = cudaEventCreateWithFlags(&c->host_step_done, cudaEventDisableTiming);
  if (e == cudaSuccess && c->host_step_recorded)
    e = cudaStreamWaitEvent(s, c->host_step_done, 0);
  if (e != cudaSuccess) return cuda_fail("kvr_decode_step_host: copy in", e);
  st = kvr_decode_step(c, lb, le, q_dev, k_new_dev, v_new_dev, out_dev, budget,
                       window, stream);
  if (st != KVR_OK) return st;
  e = cudaEventRecord(c->host_step_done, s);
  if (e == cudaSuccess) {
    c->host_step_recorded = true;
    e = cudaMemcpyAsync(out_host, out_dev, ob, cudaMemcpyDeviceToHost, s);
  }
  if (e != cudaSuccess) return cuda_fail("kvr_decode_step_host: copy out", e);
  return KVR_OK;
}

kvr_status kvr_cache_export(const kvr_cache *c, int seq, void *host_k,
                            void *host_v, float *host_score, int32_t *host_pos,
                            int32_t *host_len, int32_t *host_next_pos,
                            void *stream) {
  if (!c) return fail(KVR_EINVAL, "null cache");
  if (seq < 0 || seq >= c->desc.n_seq)
    return fail(KVR_EINVAL, "sequence %d outside [0, %d)", seq, c->desc.n_seq);
  cudaError_t e = cudaStreamSynchronize(as_stream(stream));
  if (e != cudaSuccess) return cuda_fail("kvr_cache_export: sync", e);
  const CacheView &v = c->view;
  const size_t units = (size_t)v.L * v.H, rows = units * v.cap;
  const size_t ebytes = (size_t)v.d * esize(c->desc.kv_dtype);
  struct {
    void *dst;
    const void *src;
    size_t bytes;
  } copies[] = {
      {host_k, static_cast<char *>(v.K) + seq * rows * ebytes, rows * ebytes},
      {host_v, static_cast<char *>(v.V) + seq * rows * ebytes, rows * ebytes},
  };
  for (auto &cp : copies) {
    if (!cp.dst) continue;
    e = cudaMemcpy(cp.dst, cp.src, cp.bytes, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail("kvr_cache_export", e);
  }
  // Scores and positions: [units][sstride] on the device, [units][cap] out.
  struct {
    void *dst;
    const void *src;
  } rowwise[] = {{host_score, v.score + seq * units * v.sstride},
                 {host_pos, v.pos + seq * units * v.sstride}};
  for (auto &cp : rowwise) {
    if (!cp.dst) continue;
    e = cudaMemcpy2D(cp.dst, (size_t)v.cap * 4, cp.src, (size_t)v.sstride * 4,
                     (size_t)v.cap * 4, units, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail("kvr_cache_export", e);
  }
  if (host_len || host_next_pos) {
    std::vector<int32_t> st(units * 4);
    e = cudaMemcpy(st.data(), v.state + seq * units * 4,
                   st.size() * sizeof(int32_t), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail("kvr_cache_export", e);
    for (size_t i = 0; i < units; ++i) {
      if (host_len) host_len[i] = st[4 * i];
      if (host_next_pos) host_next_pos[i] = st[4 * i + 1];
    }
  }
  return KVR_OK;
}

kvr_status kvr_cache_import(kvr_cache *c, int seq, const void *host_k,
                            const void *host_v, const float *host_score,
                            const int32_t *host_pos, const int32_t *host_len,
                            const int32_t *host_next_pos, void *stream) {
  if (!c) return fail(KVR_EINVAL, "null cache");
  if (c->forks) return fail(KVR_ESTATE, "the cache has a live fork");
  if (seq < 0 || seq >= c->desc.n_seq)
    return fail(KVR_EINVAL, "sequence %d outside [0, %d)", seq, c->desc.n_seq);
  if (!host_k || !host_v || !host_score || !host_pos || !host_len ||
      !host_next_pos)
    return fail(KVR_EINVAL, "null host buffer");
  const CacheView &v = c->view;
  const int L = v.L, H = v.H, cap = v.cap;
  std::vector<int32_t> live;
  for (int l = 0; l < L; ++l)
    for (int h = 0; h < H; ++h) {
      const size_t u = (size_t)l * H + h;
      const int n = host_len[u], np = host_next_pos[u];
      if (n < 0 || n > cap)
        return fail(KVR_EINVAL, "layer %d head %d: length %d outside [0, %d]",
                    l, h, n, cap);
      if (np < 0 || np == INT32_MAX)
        return fail(KVR_EINVAL, "layer %d head %d: next position %d", l, h, np);
      if (n != host_len[(size_t)l * H] || np != host_next_pos[(size_t)l * H])
        return fail(KVR_EINVAL,
                    "layer %d: KV heads differ in length or next position", l);
      live.assign(host_pos + u * cap, host_pos + u * cap + n);
      std::sort(live.begin(), live.end());
      for (int i = 0; i < n; ++i)
        if (live[i] < 0 || live[i] >= np || (i > 0 && live[i] == live[i - 1]))
          return fail(KVR_EINVAL,
                      "layer %d head %d: live positions must be distinct and "
                      "in [0, %d)", l, h, np);
    }
  cudaError_t e = cudaStreamSynchronize(as_stream(stream));
  if (e != cudaSuccess) return cuda_fail("kvr_cache_import: sync", e);
  const size_t units = (size_t)L * H, rows = units * cap;
  const size_t ebytes = (size_t)v.d * esize(c->desc.kv_dtype);
  e = cudaMemcpy(static_cast<char *>(v.K) + seq * rows * ebytes, host_k,
                 rows * ebytes, cudaMemcpyHostToDevice);
  if (e == cudaSuccess)
    e = cudaMemcpy(static_cast<char *>(v.V) + seq * rows * ebytes, host_v,
                   rows * ebytes, cudaMemcpyHostToDevice);
  if (e == cudaSuccess)
    e = cudaMemcpy2D(v.score + seq * units * v.sstride, (size_t)v.sstride * 4,
                     host_score, (size_t)cap * 4, (size_t)cap * 4, units,
                     cudaMemcpyHostToDevice);
  if (e == cudaSuccess)
    e = cudaMemcpy2D(v.pos + seq * units * v.sstride, (size_t)v.sstride * 4,
                     host_pos, (size_t)cap * 4, (size_t)cap * 4, units,
                     cudaMemcpyHostToDevice);
  std::vector<int32_t> st(units * 4);
  if (e == cudaSuccess)
    e = cudaMemcpy(st.data(), v.state + seq * units * 4,
                   st.size() * sizeof(int32_t), cudaMemcpyDeviceToHost);
  if (e == cudaSuccess) {
    for (size_t i = 0; i < units; ++i) {
      st[4 * i] = host_len[i];
      st[4 * i + 1] = host_next_pos[i];
      st[4 * i + 2] = 0;  // no R-KV key sum for the imported rows
    }
    e = cudaMemcpy(v.state + seq * units * 4, st.data(),
                   st.size() * sizeof(int32_t), cudaMemcpyHostToDevice);
  }
  if (e != cudaSuccess) return cuda_fail("kvr_cache_import", e);
  for (int l = 0; l < L; ++l) {
    c->len[(size_t)seq * L + l] = host_len[(size_t)l * H];
    c->next_pos[(size_t)seq * L + l] = host_next_pos[(size_t)l * H];
  }
  return KVR_OK;
}

kvr_status kvr_cache_lengths(const kvr_cache *c, int32_t *host_len) {
  if (!c || !host_len) return fail(KVR_EINVAL, "null argument");
  std::memcpy(host_len, c->len.data(), c->len.size() * sizeof(int32_t));
  return KVR_OK;
}

kvr_status kvr_cache_scores(const kvr_cache *c, float **score,
                            int32_t **pos, int32_t **state,
                            int64_t *row_stride) {
  if (!c) return fail(KVR_EINVAL, "null cache");
  if (score) *score = c->view.score;
  if (pos) *pos = c->view.pos;
  if (state) *state = c->view.state;
  if (row_stride) *row_stride = c->view.sstride;
  return KVR_OK;
}

kvr_status kvr_cache_launch_count(const kvr_cache *c, uint64_t *count) {
  if (!c || !count) return fail(KVR_EINVAL, "null argument");
  *count = c->launches;
  return KVR_OK;
}

kvr_status kvr_sync_status(kvr_cache *c, void *stream) {
  if (!c) return fail(KVR_EINVAL, "null cache");
  cudaError_t e = cudaStreamSynchronize(as_stream(stream));
  if (e != cudaSuccess) return cuda_fail("kvr_sync_status: sync", e);
  unsigned word = 0;
  e = cudaMemcpy(&word, c->view.err, sizeof word, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail("kvr_sync_status: read", e);
  if (!word) return KVR_OK;
  e = cudaMemset(c->view.err, 0, sizeof word);
  if (e != cudaSuccess) return cuda_fail("kvr_sync_status: clear", e);
  return fail(KVR_EDEVICE, "device error word 0x%x (%s%s%s%s)", word,
              word & kvr::ERR_CAPACITY ? "capacity " : "",
              word & kvr::ERR_NONFINITE ? "non-finite " : "",
              word & kvr::ERR_LENGTH ? "length " : "",
              word & kvr::ERR_TIMEOUT ? "timeout" : "");
}

const char *kvr_last_error(void) { return g_err.c_str(); }

}  // extern "C"

// ---- candidates ------------------------------------------------------------

struct kvr_fork {
  kvr_cache *parent;
  kvr::ForkView view;
  std::vector<int32_t> tlen;  // host mirror [S][L] (same for all candidates)
  int32_t *chosen_dev;        // [S]
  bool spent = false;
  bool tail_maps = false;     // TK / TV tensor maps encoded (tensor-core path)
  CUtensorMap tmTK, tmTV;     // 16-row boxes
  bool batch_maps = false;    // 3-D tail maps (candidate-batched kernel)
  CUtensorMap tmTK3, tmTV3;
  // Tail maps of the tensor-memory kernel, per tail length nt (encoded on
  // first use): 0 not yet, 1 encoded, -1 cannot be encoded.
  std::vector<signed char> tc_state;
  std::vector<std::array<CUtensorMap, 2>> tc_tails;
  int kernel = 0;             // kvr_fork_set_kernel choice
  int last_kernel = 0;        // the kernel that ran the last step (1..5)
};

namespace {

struct ForkLayout {
  size_t pscore, tk, tv, tscore, tpos, tlen, chosen, total;
};

ForkLayout fork_layout(const kvr_cache *p, int n_cand, int tail_cap) {
  const kvr_cache_desc &d = p->desc;
  const size_t units = (size_t)d.n_seq * d.n_layers * d.n_kv_heads;
  const size_t cu = units * (size_t)n_cand;
  const size_t tstride = kvr::round_up16(tail_cap);
  ForkLayout l{};
  size_t off = 0;
  l.pscore = off;
  off = align_up(off + cu * kvr::round_up16(d.capacity) * sizeof(float));
  l.tk = off;
  off = align_up(off + cu * tail_cap * d.head_dim * esize(d.kv_dtype));
  l.tv = off;
  off = align_up(off + cu * tail_cap * d.head_dim * esize(d.kv_dtype));
  l.tscore = off;
  off = align_up(off + cu * tstride * sizeof(float));
  l.tpos = off;
  off = align_up(off + cu * tstride * sizeof(int32_t));
  l.tlen = off;
  off = align_up(off + cu * sizeof(int32_t));
  l.chosen = off;
  off = align_up(off + (size_t)d.n_seq * sizeof(int32_t));
  l.total = off;
  return l;
}

bool fork_args_ok(const kvr_cache *p, int n_cand, int tail_cap) {
  return p && n_cand >= 1 && n_cand <= 64 && tail_cap >= 1 &&
         tail_cap <= (1 << 20);
}

kvr_status check_fork(const kvr_fork *f) {
  if (!f) return fail(KVR_EINVAL, "null fork");
  if (f->spent) return fail(KVR_ESTATE, "the fork has been committed");
  return KVR_OK;
}

}  // namespace

extern "C" {

size_t kvr_fork_required_bytes(const kvr_cache *parent, int n_cand,
                               int tail_cap) {
  if (!fork_args_ok(parent, n_cand, tail_cap)) return 0;
  return fork_layout(parent, n_cand, tail_cap).total;
}

kvr_status kvr_fork_candidates(kvr_cache *p, int n_cand, int tail_cap,
                               void *dev_buf, size_t bytes, void *stream,
                               kvr_fork **out) {
  if (!out) return fail(KVR_EINVAL, "null output handle");
  *out = nullptr;
  if (!fork_args_ok(p, n_cand, tail_cap))
    return fail(KVR_EINVAL, "bad fork arguments (%d candidates, tail %d)",
                n_cand, tail_cap);
  if (p->forks) return fail(KVR_ESTATE, "the cache already has a live fork");
  if (!dev_buf || reinterpret_cast<uintptr_t>(dev_buf) % kAlign)
    return fail(KVR_EINVAL, "null or unaligned fork buffer");
  const ForkLayout lay = fork_layout(p, n_cand, tail_cap);
  if (bytes < lay.total)
    return fail(KVR_ENOMEM, "fork buffer of %zu bytes < required %zu", bytes,
                lay.total);
  kvr_fork *f = new (std::nothrow) kvr_fork();
  if (!f) return fail(KVR_ENOMEM, "host allocation failed");
  char *b = static_cast<char *>(dev_buf);
  kvr::ForkView &v = f->view;
  v.p = p->view;
  v.N = n_cand;
  v.tcap = tail_cap;
  v.tstride = kvr::round_up16(tail_cap);
  v.pscore = reinterpret_cast<float *>(b + lay.pscore);
  v.TK = b + lay.tk;
  v.TV = b + lay.tv;
  v.tscore = reinterpret_cast<float *>(b + lay.tscore);
  v.tpos = reinterpret_cast<int32_t *>(b + lay.tpos);
  v.tlen = reinterpret_cast<int32_t *>(b + lay.tlen);
  f->chosen_dev = reinterpret_cast<int32_t *>(b + lay.chosen);
  f->parent = p;
  f->tlen.assign(p->len.size(), 0);
  const size_t units =
      (size_t)p->desc.n_seq * p->desc.n_layers * p->desc.n_kv_heads;
  const size_t sbytes = units * p->view.sstride * sizeof(float);
  cudaStream_t st = as_stream(stream);
  cudaError_t e = cudaSuccess;
  for (int c = 0; c < n_cand && e == cudaSuccess; ++c)
    e = cudaMemcpyAsync(v.pscore + c * units * p->view.sstride, p->view.score,
                        sbytes, cudaMemcpyDeviceToDevice, st);
  if (e == cudaSuccess)
    e = cudaMemsetAsync(v.tlen, 0, units * n_cand * sizeof(int32_t), st);
  if (e != cudaSuccess) {
    delete f;
    return cuda_fail("kvr_fork_candidates", e);
  }
  if (p->view.kv_bf16 && p->view.d == 128 &&
      (size_t)n_cand * units * tail_cap < (size_t)INT32_MAX) {
    const size_t trows = (size_t)n_cand * units * tail_cap;
    f->tail_maps =
        encode_slab(&f->tmTK, v.TK, trows, kvr::fork_mma_box_rows()) &&
        encode_slab(&f->tmTV, v.TV, trows, kvr::fork_mma_box_rows());
    const int T = kvr::fork_batch_tail_rows(n_cand);
    f->batch_maps =
        T > 0 &&
        encode_tails3(&f->tmTK3, v.TK, units * (size_t)tail_cap, n_cand, T) &&
        encode_tails3(&f->tmTV3, v.TV, units * (size_t)tail_cap, n_cand, T);
    f->tc_state.assign(std::min(tail_cap, kvr::fork_tc_max_tail()) + 1, 0);
    f->tc_tails.resize(f->tc_state.size());
  }
  p->forks += 1;
  *out = f;
  return KVR_OK;
}

kvr_status kvr_fork_decode_attend_score(kvr_fork *f, int lb, int le,
                                        const void *q, const void *k_new,
                                        const void *v_new, void *out,
                                        void *stream) {
  kvr_status st = check_fork(f);
  if (st != KVR_OK) return st;
  kvr_cache *p = f->parent;
  st = check_layers(p, lb, le);
  if (st != KVR_OK) return st;
  if (!q || !k_new || !v_new || !out)
    return fail(KVR_EINVAL, "null q, k_new, v_new or out");
  int max_prefix = 0, n_max = 0;
  for (int s = 0; s < p->desc.n_seq; ++s)
    for (int l = lb; l < le; ++l) {
      const size_t i = (size_t)s * p->desc.n_layers + l;
      if (f->tlen[i] + 1 > f->view.tcap)
        return fail(KVR_ECAPACITY, "a candidate tail holds %d rows; capacity %d"
                    " is full", f->tlen[i], f->view.tcap);
      max_prefix = std::max(max_prefix, p->len[i]);
      n_max = std::max(n_max, p->len[i] + f->tlen[i] + 1);
    }
  int dev = 0, optin = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  if (kvr::fork_attend_smem_bytes(p->view, n_max, max_prefix) > (size_t)optin)
    return fail(KVR_EINVAL, "prefix of %d rows is too long for the candidate "
                "kernel's shared memory", max_prefix);
  StepArgs a{};
  a.lb = lb;
  a.nl = le - lb;
  a.q = q;
  a.k_new = k_new;
  a.v_new = v_new;
  a.out = out;
  a.max_rows = n_max;
  cudaError_t e = cudaSuccess;
  int nt_max = 0;
  for (int s = 0; s < p->desc.n_seq; ++s)
    for (int l = lb; l < le; ++l)
      nt_max = std::max(nt_max, f->tlen[(size_t)s * p->desc.n_layers + l]);
  const CacheView &pv = p->view;
  const std::pair<CUtensorMap, CUtensorMap> *maps = nullptr, *maps128 = nullptr;
  const int want = p->fused ? f->kernel : 4;  // 0 auto, 1..5 one kernel
  // The tensor-memory kernel (chosen explicitly only: the candidate-batched
  // kernel is faster at the sizes measured) wants every unit of the call at
  // the same tail length (its tail maps end there).
  bool nt_same = true;
  for (int s = 0; s < p->desc.n_seq && nt_same; ++s)
    for (int l = lb; l < le; ++l)
      nt_same = nt_same && f->tlen[(size_t)s * p->desc.n_layers + l] == nt_max;
  const CUtensorMap *tails = nullptr;
  if (want == 5 && nt_same && (size_t)nt_max < f->tc_state.size()) {
    signed char &st8 = f->tc_state[nt_max];
    if (st8 == 0) {
      const size_t units = (size_t)pv.S * pv.L * pv.H;
      const int rows = std::max(nt_max, 1);
      st8 = encode_tails4(&f->tc_tails[nt_max][0], f->view.TK, rows, f->view.tcap, units,
                          f->view.N) &&
                    encode_tails4(&f->tc_tails[nt_max][1], f->view.TV, rows, f->view.tcap,
                                  units, f->view.N)
                ? 1
                : -1;
    }
    if (st8 == 1) tails = f->tc_tails[nt_max].data();
  }
  const bool tc_ok =
      want == 5 && p->fused && tails && pv.G <= 8 &&
      f->view.N <= kvr::fork_tc_max_cand() && device_facts(p) &&
      kvr::fork_tc_smem_bytes() <= (size_t)p->smem_optin &&
      max_prefix <= kvr::fork_tc_max_prefix() && nt_max <= kvr::fork_tc_max_tail() &&
      (size_t)pv.S * pv.L * pv.H * pv.cap < (size_t)INT32_MAX &&
      aligned16(q) && aligned16(k_new) && aligned16(v_new) && aligned16(out) &&
      (maps = slab_maps(p, kvr::fork_tc_box_rows())) != nullptr;
  const bool batch_ok = !tc_ok &&
      (want == 0 || want == 1) && p->fused && f->batch_maps && pv.G <= 8 &&
      f->view.N <= kvr::fork_batch_max_cand() && device_facts(p) &&
      kvr::fork_batch_smem_bytes(n_max, f->view.N) + 512 <=
          (size_t)p->smem_optin &&
      (size_t)pv.S * pv.L * pv.H * pv.cap < (size_t)INT32_MAX &&
      aligned16(q) && aligned16(k_new) && aligned16(v_new) && aligned16(out) &&
      (maps = slab_maps(p, kvr::chunk_box_rows())) != nullptr &&
      (maps128 = slab_maps(p, kvr::fork_batch_prefix_box_rows())) != nullptr;
  kvr::ChunkParams cp{};
  const bool chunk_ok = !batch_ok && (want == 0 || want == 2) &&
      p->fused && p->chunk_groups >= 0 && f->tail_maps && pv.G <= 8 &&
      n_max <= kvr::chunk_max_rows() && device_facts(p) &&
      chunk_config(p, n_max, &cp.n_groups, &cp.n_stages) &&
      (size_t)pv.S * pv.L * pv.H * pv.cap < (size_t)INT32_MAX &&
      aligned16(q) && aligned16(k_new) && aligned16(v_new) && aligned16(out) &&
      (maps = slab_maps(p, kvr::chunk_box_rows())) != nullptr;
  const bool mma_ok = !batch_ok && !chunk_ok && (want == 0 || want == 3) &&
      p->fused && f->tail_maps && pv.G <= 8 &&
      f->view.N <= kvr::fork_mma_max_cand() && device_facts(p) &&
      kvr::fork_mma_smem_bytes(max_prefix, nt_max, f->view.N) + 512 <=
          (size_t)p->smem_optin &&
      (size_t)pv.S * pv.L * pv.H * pv.cap < (size_t)INT32_MAX &&
      aligned16(q) && aligned16(k_new) && aligned16(v_new) && aligned16(out) &&
      (maps = slab_maps(p, kvr::fork_mma_box_rows())) != nullptr;
  if (tc_ok) {
    kvr::ForkTcParams tp{};
    tp.f = f->view;
    tp.q = static_cast<const __nv_bfloat16 *>(q);
    tp.k_new = static_cast<const __nv_bfloat16 *>(k_new);
    tp.v_new = static_cast<const __nv_bfloat16 *>(v_new);
    tp.out = out;
    tp.lb = lb;
    tp.nl = le - lb;
    tp.scale_log2e = pv.scale * 1.4426950408889634f;
    tp.inv_g = 1.f / (float)pv.G;
    const int units = pv.S * (le - lb) * pv.H;
    tp.nt = nt_max;
    tp.np_max = max_prefix;
    e = kvr::launch_fork_tc(maps->first, maps->second, &tails[0], &tails[1], tp,
                            std::min(p->sm_count, units), as_stream(stream));
  } else if (batch_ok) {
    kvr::ForkBatchParams bp{};
    bp.f = f->view;
    bp.q = static_cast<const __nv_bfloat16 *>(q);
    bp.k_new = static_cast<const __nv_bfloat16 *>(k_new);
    bp.v_new = static_cast<const __nv_bfloat16 *>(v_new);
    bp.out = out;
    bp.lb = lb;
    bp.nl = le - lb;
    bp.n_max = n_max;
    bp.scale_log2e = pv.scale * 1.4426950408889634f;
    bp.inv_g = 1.f / (float)pv.G;
    const int units = pv.S * (le - lb) * pv.H;
    e = kvr::launch_fork_batch(maps->first, maps->second, maps128->first,
                               maps128->second, f->tmTK3, f->tmTV3, bp,
                               std::min(p->sm_count, units), as_stream(stream));
  } else if (chunk_ok) {
    cp.c = pv;
    cp.f = f->view;
    cp.fork = 1;
    cp.q = static_cast<const __nv_bfloat16 *>(q);
    cp.k_new = static_cast<const __nv_bfloat16 *>(k_new);
    cp.v_new = static_cast<const __nv_bfloat16 *>(v_new);
    cp.out = out;
    cp.lb = lb;
    cp.nl = le - lb;
    cp.n_jobs = f->view.N * pv.S * (le - lb) * pv.H;
    cp.n_max = n_max;
    cp.scale_log2e = pv.scale * 1.4426950408889634f;
    cp.inv_g = 1.f / (float)pv.G;
    const int grid = std::min(p->sm_count, cp.n_jobs);
    e = kvr::launch_chunk_step(maps->first, maps->second, &f->tmTK, &f->tmTV,
                               cp, grid, as_stream(stream));
  } else if (mma_ok) {
    kvr::ForkMmaParams mp{};
    mp.f = f->view;
    mp.q = static_cast<const __nv_bfloat16 *>(q);
    mp.k_new = static_cast<const __nv_bfloat16 *>(k_new);
    mp.v_new = static_cast<const __nv_bfloat16 *>(v_new);
    mp.out = out;
    mp.lb = lb;
    mp.nl = le - lb;
    mp.np_max = max_prefix;
    mp.nt_max = nt_max;
    mp.scale_log2e = pv.scale * 1.4426950408889634f;
    e = kvr::launch_fork_mma(maps->first, maps->second, f->tmTK, f->tmTV, mp,
                             as_stream(stream));
  } else {
    e = kvr::launch_fork_attend(f->view, a, n_max, max_prefix,
                                as_stream(stream));
  }
  if (e != cudaSuccess) return cuda_fail("kvr_fork_decode_attend_score", e);
  f->last_kernel = tc_ok ? 5 : batch_ok ? 1 : chunk_ok ? 2 : mma_ok ? 3 : 4;
  p->launches += 1;
  for (int s = 0; s < p->desc.n_seq; ++s)
    for (int l = lb; l < le; ++l) f->tlen[(size_t)s * p->desc.n_layers + l] += 1;
  return KVR_OK;
}

kvr_status kvr_fork_commit(kvr_fork *f, const int32_t *chosen, int budget,
                           int window, void *stream) {
  kvr_status st = check_fork(f);
  if (st != KVR_OK) return st;
  if (!chosen) return fail(KVR_EINVAL, "null chosen");
  st = check_evict(budget, window);
  if (st != KVR_OK) return st;
  kvr_cache *p = f->parent;
  for (int s = 0; s < p->desc.n_seq; ++s)
    if (chosen[s] < 0 || chosen[s] >= f->view.N)
      return fail(KVR_EINVAL, "chosen[%d] = %d outside [0, %d)", s, chosen[s],
                  f->view.N);
  int max_rows = 1;
  for (size_t i = 0; i < p->len.size(); ++i)
    max_rows = std::max(max_rows, p->len[i] + f->tlen[i]);
  cudaStream_t strm = as_stream(stream);
  cudaError_t e = cudaMemcpyAsync(f->chosen_dev, chosen,
                                  p->desc.n_seq * sizeof(int32_t),
                                  cudaMemcpyHostToDevice, strm);
  if (e == cudaSuccess)
    e = kvr::launch_fork_commit(f->view, f->chosen_dev, max_rows, budget,
                                window, strm);
  if (e != cudaSuccess) return cuda_fail("kvr_fork_commit", e);
  p->launches += 1;
  for (size_t i = 0; i < p->len.size(); ++i) {
    p->len[i] = (int32_t)std::min<long long>((long long)p->len[i] + f->tlen[i],
                                             (long long)budget + window);
    p->next_pos[i] += f->tlen[i];
  }
  f->spent = true;
  p->forks -= 1;
  return KVR_OK;
}

kvr_status kvr_fork_export(const kvr_fork *f, int cand, int seq,
                           float *host_prefix_score, void *host_tail_k,
                           void *host_tail_v, float *host_tail_score,
                           int32_t *host_tail_pos, int32_t *host_tail_len,
                           void *stream) {
  if (!f) return fail(KVR_EINVAL, "null fork");
  const kvr_cache *p = f->parent;
  const kvr::ForkView &v = f->view;
  if (cand < 0 || cand >= v.N || seq < 0 || seq >= p->desc.n_seq)
    return fail(KVR_EINVAL, "candidate %d / sequence %d out of range", cand,
                seq);
  cudaError_t e = cudaStreamSynchronize(as_stream(stream));
  if (e != cudaSuccess) return cuda_fail("kvr_fork_export: sync", e);
  const size_t units =
      (size_t)p->desc.n_seq * p->desc.n_layers * p->desc.n_kv_heads;
  const size_t per_seq = (size_t)p->desc.n_layers * p->desc.n_kv_heads;
  const size_t cu0 = (size_t)cand * units + (size_t)seq * per_seq;
  const size_t ebytes = (size_t)p->desc.head_dim * esize(p->desc.kv_dtype);
  if (host_prefix_score &&
      (e = cudaMemcpy2D(host_prefix_score, (size_t)p->view.cap * 4,
                        v.pscore + cu0 * p->view.sstride,
                        (size_t)p->view.sstride * 4, (size_t)p->view.cap * 4,
                        per_seq, cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail("kvr_fork_export", e);
  const size_t tbytes = per_seq * v.tcap * ebytes;
  if (host_tail_k &&
      (e = cudaMemcpy(host_tail_k,
                      static_cast<char *>(v.TK) + cu0 * v.tcap * ebytes, tbytes,
                      cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail("kvr_fork_export", e);
  if (host_tail_v &&
      (e = cudaMemcpy(host_tail_v,
                      static_cast<char *>(v.TV) + cu0 * v.tcap * ebytes, tbytes,
                      cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail("kvr_fork_export", e);
  if (host_tail_score &&
      (e = cudaMemcpy2D(host_tail_score, (size_t)v.tcap * 4,
                        v.tscore + cu0 * v.tstride, (size_t)v.tstride * 4,
                        (size_t)v.tcap * 4, per_seq,
                        cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail("kvr_fork_export", e);
  if (host_tail_pos &&
      (e = cudaMemcpy2D(host_tail_pos, (size_t)v.tcap * 4,
                        v.tpos + cu0 * v.tstride, (size_t)v.tstride * 4,
                        (size_t)v.tcap * 4, per_seq,
                        cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail("kvr_fork_export", e);
  if (host_tail_len &&
      (e = cudaMemcpy(host_tail_len, v.tlen + cu0, per_seq * sizeof(int32_t),
                      cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail("kvr_fork_export", e);
  return KVR_OK;
}

int kvr_fork_last_kernel(const kvr_fork *f) { return f ? f->last_kernel : 0; }

int kvr_cache_last_absorb_kernel(const kvr_cache *c) { return c ? c->last_absorb : -1; }

kvr_status kvr_fork_set_kernel(kvr_fork *f, int kernel) {
  if (!f) return fail(KVR_EINVAL, "null fork");
  if (kernel < 0 || kernel > 5)
    return fail(KVR_EINVAL, "fork kernel %d outside [0, 5]", kernel);
  f->kernel = kernel;
  return KVR_OK;
}

void kvr_fork_destroy(kvr_fork *f) {
  if (!f) return;
  if (!f->spent) f->parent->forks -= 1;
  delete f;
}

}  // extern "C"
