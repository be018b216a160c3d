// kvr_internal.h -- shared between the C-ABI host code and the kernels of
// libkvr.  Not installed; not part of the ABI.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace kvr {

// Device error word bits (set with atomicOr, read by kvr_sync_status).
enum : unsigned {
  ERR_CAPACITY = 1u,   // a unit had no free row for the append
  ERR_NONFINITE = 2u,  // a softmax normaliser was not finite
  ERR_LENGTH = 4u,     // an eviction produced an unexpected live length
  ERR_TIMEOUT = 8u,    // a bounded wait on an asynchronous copy gave up
};

__host__ __device__ inline int round_up16(int x) { return (x + 15) & ~15; }

// Every kernel of libkvr is launched with programmatic stream serialization
// (launch_pdl): it may start while the previous kernel of the stream drains,
// so it runs pdl_begin() before its first global memory access.  The wait
// returns once the previous grid has completed and its writes are visible;
// the trigger then lets the next launch start early in turn.
__device__ __forceinline__ void pdl_begin() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block,
                       size_t smem, cudaStream_t st, Args &&...args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<Args &&>(args)...);
}

// Default bound of a step kernel's wait on an asynchronous copy (2 s).
constexpr unsigned long long kDefaultWaitNs = 2000000000ull;

// Device view of one cache: every pointer points into the caller's buffer.
// A unit u = (s * L + l) * H + h.
struct CacheView {
  void *K;          // [u][cap][d] kv element type
  void *V;          // [u][cap][d]
  float *score;     // [u][sstride]
  int32_t *pos;     // [u][sstride]
  int32_t *state;   // [u][4]: live length, next position, rsum valid, 0
  unsigned *err;    // device error word
  float *logits;    // [u][G][cap] scratch for units beyond on-chip size
  float *rsum;      // [u][d] R-KV: sum of the live rows' normalised keys,
                    // kept by kvr_decode_step_rkv's one-launch step; valid
                    // while the unit's state word 2 is 1 (every other call
                    // that changes the unit's rows writes 0 there)
  int S, L, H, G, d, cap;
  int sstride;      // cap rounded up to 16 (64-byte aligned score/pos rows)
  float scale;      // softmax scale (1/sqrt(d) by default)
  int kv_bf16;      // 1: bf16 elements, 0: fp32
  int out_bf16;     // 1: bf16 output, 0: fp32
  // Bound of the step kernels' waits on this cache's asynchronous copies
  // (kvr_cache_set_wait_limit; 2 s by default).
  unsigned long long wait_ns;
  // Test hook (kvr_cache_set_hold_first_unit): the fused and chunked step
  // kernels never load the first unit of CTA 0, so its consumers' bounded
  // wait runs out and the launch ends with ERR_TIMEOUT.
  int hold_first;
};

// Work description of one decode call over layers [lb, lb + nl).
struct StepArgs {
  int lb, nl;
  const void *q;      // [S][nl][H*G][d]
  const void *k_new;  // [S][nl][H][d]
  const void *v_new;  // [S][nl][H][d]
  void *out;          // [S][nl][H*G][d]
  int max_rows;       // largest live length after the append over the units
  int budget, window; // eviction target (evict only when evict != 0)
  int evict;
  // Inputs holding `chunk` tokens per (sequence, layer) row, [S][nl][chunk]
  // [...] (kvr_absorb_chunk); this call reads token `tok` of each.
  int chunk = 1, tok = 0;
};

// Generic kernels (any d in {64,128}, G <= 8, fp32 or bf16): one CTA per unit.
cudaError_t launch_attend_score_generic(const CacheView &c, const StepArgs &a,
                                        cudaStream_t st);
// The attend kernel with its logits always in `ext` (one [G][max_rows] fp32
// block per (sequence, layer, KV head) of the launch, in launch order).
cudaError_t launch_attend_score_ext_scratch(const CacheView &c,
                                            const StepArgs &a, float *ext,
                                            cudaStream_t st);
// Eviction with the R-KV score (mix weight lam in [0, 1]); the z of each
// unit's rows is kept in its logit scratch.
cudaError_t launch_evict_rkv(const CacheView &c, int lb, int nl, int max_rows,
                             int budget, int window, float lam,
                             cudaStream_t st);
cudaError_t launch_evict_generic(const CacheView &c, int lb, int nl,
                                 int max_rows, int budget, int window,
                                 cudaStream_t st);
cudaError_t launch_load(const CacheView &c, int seq, const void *k,
                        const void *v, int n_rows, int first_pos,
                        cudaStream_t st);
cudaError_t launch_init(const CacheView &c, cudaStream_t st);

// Sequence pairs of one kvr_cache_copy_sequences launch (passed by value).
constexpr int kMaxSeqPairs = 1024;
struct SeqPairs {
  int32_t src[kMaxSeqPairs];
  int32_t dst[kMaxSeqPairs];
};
// Copy the whole state of sequence p.src[i] of `src` into sequence p.dst[i]
// of `dst`, i < n_pairs <= kMaxSeqPairs; row_bytes = d * element size.
cudaError_t launch_copy_seqs(const CacheView &dst, const CacheView &src,
                             const SeqPairs &p, int n_pairs, int row_bytes,
                             cudaStream_t st);

// Fused steady-state step (kvr_fused.cu): bf16, d = 128, G <= 8, at most 160
// live rows per unit after the append, at most one eviction per unit.
struct FusedParams {
  CacheView c;
  const __nv_bfloat16 *q;      // [S][nl][H*G][128]
  const __nv_bfloat16 *k_new;  // [S][nl][H][128]
  const __nv_bfloat16 *v_new;  // [S][nl][H][128]
  void *out;                   // [S][nl][H*G][128]
  int lb, nl;
  int R;                       // staged rows per unit (multiple of 16, <= 128)
  int Rb;                      // rows copied from a slab (multiple of 8, <= R)
  int n_stages, n_groups;      // ring depth; units computed at once
  int group_warps;             // warps sharing one unit
  int budget, window, evict;
  float scale_log2e, inv_g;
  // R-KV eviction (App. C) instead of the accumulated-attention TopB: the
  // evicted row is the candidate of lowest z = lam * I - (1 - lam) * R.
  int rkv;
  float lam;
};
int fused_stage_bytes(int R, bool rkv = false);
// Warps that share one unit of R staged rows: `requested` if it is one of
// the supported choices (one or two row tiles per warp), else the default.
int fused_group_warps(int R, int requested);
// Bytes of one consumer group's exchange area (after the ring of stages);
// the R-KV step needs one more statistics slot a warp.
int fused_group_bytes(int U, bool rkv = false);
int fused_max_groups();
int fused_max_rows();   // live rows a unit after the append (160)
int fused_max_threads();
int fused_producer_warps();
cudaError_t launch_fused_step(const CUtensorMap &tmK, const CUtensorMap &tmV,
                              const FusedParams &p, int grid, int smem_bytes,
                              cudaStream_t st);

// Fused step for longer units (kvr_stream.cu): bf16, d = 128, G <= 8, at
// most stream_max_rows() rows after the append, at most one eviction.
struct StreamParams {
  CacheView c;
  const __nv_bfloat16 *q, *k_new, *v_new;
  void *out;
  int lb, nl;
  int n_max;                   // largest live length after the append
  int budget, window, evict;
  float scale_log2e;
};
int stream_box_rows();
int stream_max_rows();
size_t stream_smem_bytes(int n_max);
cudaError_t launch_stream_step(const CUtensorMap &tmK, const CUtensorMap &tmV,
                               const StreamParams &p, cudaStream_t st);

// Full-context decode split over the rows (kvr_split.cu): bf16, d = 128,
// G <= 8.  ws holds [units of the call][n_splits][G][130] floats.
struct SplitParams {
  CacheView c;
  const __nv_bfloat16 *q, *k_new, *v_new;
  int lb, nl, n_splits;
  float *ws;
  float scale_log2e;
};
size_t split_workspace_bytes(const CacheView &c, int nl, int n_splits);
int split_rows_per_stage();
cudaError_t launch_split_attend(const CUtensorMap &tmK, const CUtensorMap &tmV,
                                const SplitParams &p, void *out,
                                cudaStream_t st);

// Candidates of one cache (kvr_fork.cu).  A candidate unit cu = c * units + u.
struct ForkView {
  CacheView p;       // the parent: its live rows are every candidate's prefix
  int N;             // candidates
  int tcap;          // tail rows per candidate unit
  int tstride;       // tcap rounded up to 16
  float *pscore;     // [N][units][p.sstride] candidate copies of the scores
  void *TK, *TV;     // [N][units][tcap][d]
  float *tscore;     // [N][units][tstride]
  int32_t *tpos;     // [N][units][tstride]
  int32_t *tlen;     // [N][units]
};
size_t fork_attend_smem_bytes(const CacheView &c, int n_max, int max_prefix);

// Candidate step on tensor cores (kvr_fork_mma.cu): bf16, d = 128, G <= 8,
// N <= fork_mma_max_cand(); one CTA per unit, one warp per candidate.
struct ForkMmaParams {
  ForkView f;
  const __nv_bfloat16 *q, *k_new, *v_new;  // [N][S][nl][...][128]
  void *out;
  int lb, nl;
  int np_max;   // longest prefix over the call's units
  int nt_max;   // longest tail (before the append) over the call's units
  float scale_log2e;
};
size_t fork_mma_smem_bytes(int np_max, int nt_max, int n_cand);
int fork_mma_box_rows();
int fork_mma_max_cand();
cudaError_t launch_fork_mma(const CUtensorMap &tmK, const CUtensorMap &tmV,
                            const CUtensorMap &tmTK, const CUtensorMap &tmTV,
                            const ForkMmaParams &p, cudaStream_t st);
cudaError_t launch_fork_attend(const ForkView &f, const StepArgs &a, int n_max,
                               int max_prefix, cudaStream_t st);
cudaError_t launch_fork_commit(const ForkView &f, const int32_t *chosen,
                               int max_rows, int budget, int window,
                               cudaStream_t st);

// Candidate-batched step (kvr_fork_batch.cu): bf16, d = 128, G <= 8,
// N <= fork_batch_max_cand(); persistent CTAs, a warp per candidate, the
// parent's rows streamed once per unit for all candidates.
struct ForkBatchParams {
  ForkView f;
  const __nv_bfloat16 *q, *k_new, *v_new;  // [N][S][nl][...][128]
  void *out;
  int lb, nl;
  int n_max;   // largest prefix + tail + 1 over the call's units
  float scale_log2e, inv_g;
};
int fork_batch_max_cand();
// Box heights of the maps it takes: the parent slab in 16-row boxes and in
// fork_batch_prefix_box_rows()-row boxes (a full prefix block); the tails as
// a 3-D map {128, units * tcap, N} with boxes {64, fork_batch_tail_rows(N), N}.
int fork_batch_prefix_box_rows();
int fork_batch_tail_rows(int n_cand);
size_t fork_batch_smem_bytes(int n_max, int n_cand);
cudaError_t launch_fork_batch(const CUtensorMap &tmK, const CUtensorMap &tmV,
                              const CUtensorMap &tmK128,
                              const CUtensorMap &tmV128,
                              const CUtensorMap &tmTK, const CUtensorMap &tmTV,
                              const ForkBatchParams &p, int grid,
                              cudaStream_t st);

// Candidate step on 5th-generation tensor cores (kvr_fork_tc.cu): bf16,
// d = 128, G <= 8, N <= fork_tc_max_cand(), at most fork_tc_max_prefix()
// parent rows and fork_tc_max_tail() tail rows (before the append) per unit;
// one persistent CTA per SM with two units in flight; every unit of the call
// holds nt tail rows.  It takes the parent slab maps with
// fork_tc_box_rows()-row boxes and the tails as 4-D maps {128, max(nt, 1),
// units, N} (strides 256 B, tcap rows, units * tcap rows) with boxes {64,
// nt rounded up to 16, 1, min(N, 2)}.
struct ForkTcParams {
  ForkView f;
  const __nv_bfloat16 *q, *k_new, *v_new;  // [N][S][nl][...][128]
  void *out;
  int lb, nl;
  int nt;      // tail rows before the append, the same in every unit
  int np_max;  // largest prefix (parent rows) over the call's units
  float scale_log2e, inv_g;
};
int fork_tc_max_cand();
int fork_tc_max_prefix();
int fork_tc_max_tail();
int fork_tc_box_rows();
size_t fork_tc_smem_bytes();
cudaError_t launch_fork_tc(const CUtensorMap &tmK, const CUtensorMap &tmV,
                           const CUtensorMap *tmTK, const CUtensorMap *tmTV,
                           const ForkTcParams &p, int grid, cudaStream_t st);

// Absorbing a chunk of tokens (kvr_absorb.cu): bf16, d = 128, G <= 8,
// chunk <= absorb_max_chunk(), at most absorb_max_rows() rows after it.
struct AbsorbParams {
  CacheView c;
  const __nv_bfloat16 *q, *k_new, *v_new;  // [S][nl][chunk][...][128]
  void *out;
  int lb, nl, chunk;
  int max_rows;  // largest unit after the chunk over the call
  int budget, window, evict;
  float scale_log2e, inv_g;
};
int absorb_max_chunk();
int absorb_max_rows();
// kernel: 0 the tensor-memory (tcgen05) kernel (units of at most 144 rows
// after the chunk, given tmQ; otherwise the other), 1 the mma.sync kernel.
// tmQ: q as a 4-D tensor {128, G, H, S * nl * chunk tokens} with boxes
// {64, G, 1, 128 / G} and 128-byte swizzle.
// *ran (if given): the kernel launched, 0 tcgen05 or 1 mma.sync.
cudaError_t launch_absorb(const AbsorbParams &p, int kernel, const CUtensorMap *tmQ,
                          cudaStream_t st, int *ran = nullptr);

// Persistent chunked step (kvr_chunked.cu): bf16, d = 128, G <= 8, at most
// chunk_max_rows() rows per job with the new row.  A job is one unit of the
// cache (fork == 0: its live rows, the new row, at most one eviction) or one
// candidate of one unit (fork == 1: the parent's live rows as a read-only
// prefix, the candidate's tail, the new row appended to the tail).
struct ChunkParams {
  CacheView c;
  ForkView f;                  // fork == 1 only
  int fork;
  const __nv_bfloat16 *q, *k_new, *v_new;  // [jobs' rows][...][128]
  void *out;
  int lb, nl;
  int n_jobs;                  // S * nl * H, times N for candidates
  int n_max;                   // largest job (rows with the new row)
  int n_groups, n_stages;      // consumer groups; ring stages per group
  int budget, window, evict;
  float scale_log2e, inv_g;
};
int chunk_box_rows();
int chunk_max_rows();
int chunk_max_groups();
int chunk_max_stages();
size_t chunk_smem_bytes(int n_max, int n_groups, int n_stages);
cudaError_t launch_chunk_step(const CUtensorMap &tmK, const CUtensorMap &tmV,
                              const CUtensorMap *tmTK, const CUtensorMap *tmTV,
                              const ChunkParams &p, int grid, cudaStream_t st);

}  // namespace kvr

struct kvr_cache;
namespace kvr {
// kvr_decode_attend_score with the logit scratch supplied by the caller of
// this internal function (ext, ext_floats) instead of the cache buffer.
int decode_attend_score_ext(kvr_cache *c, int lb, int le, const void *q,
                            const void *k_new, const void *v_new, void *out,
                            float *ext, size_t ext_floats, void *stream);
// Record a CUDA failure as the thread's last error; returns KVR_ECUDA.
int report_cuda_error(const char *where, cudaError_t e);
// Record msg as the thread's last error; returns st.
int report_error(int st, const char *msg);
}  // namespace kvr
