// kernels.cuh — internal launch interface between the C ABI (api.cu) and the
// kernels.  Not installed; callers use include/ssd.h.
#pragma once

#include "common.cuh"

namespace ssd {

// Frontier size (Sec. 3.3) after n_c committed grid tokens: the horizontal
// part completes the current grid row (at most k_h positions when k_h > 0),
// and when it does, the k_v rows below follow, clipped at the last grid row;
// one contiguous raster run.
__device__ __forceinline__ int32_t frontier_size(const ssd_grid& g, int32_t n_c) {
  const int32_t y0 = n_c / g.grid_w;
  const int32_t c = n_c - y0 * g.grid_w;
  if (y0 >= g.grid_h) return 0;
  const int32_t h = g.k_h > 0 ? min(g.k_h, g.grid_w - c) : g.grid_w - c;
  const int32_t rows_below = (c + h == g.grid_w) ? min(g.k_v, g.grid_h - 1 - y0) : 0;
  return h + rows_below * g.grid_w;
}

// Drafts of a sequence with cache length `cache_len` (its positions are
// n_c .. n_c + n - 1, n_c = cache_len - prefix_len), or -1 when cache_len is
// outside the grid or the frontier does not fit D_max (reported by the caller).
__device__ __forceinline__ int32_t frontier_drafts(const ssd_grid& g, int32_t cache_len,
                                                   int32_t D_max) {
  const int32_t n_c = cache_len - g.prefix_len;
  if (n_c < 0 || n_c > g.grid_h * g.grid_w) return -1;
  const int32_t n = frontier_size(g, n_c);
  return n > D_max ? -1 : n;  // the host checks D_max >= (k_v + 1) W; keep the guard
}

// Launch `kernel`, optionally as a programmatic dependent of the kernel
// before it on `stream` (cudaLaunchAttributeProgrammaticStreamSerialization).
template <typename... KArgs, typename... Args>
cudaError_t launch_kernel(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                          cudaStream_t stream, bool pdl, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

// ---- frontier.cu
cudaError_t launch_record_commit(int32_t B, int32_t D_max, int32_t prefix_len, int32_t hw,
                                 const int32_t* cache_len, const int32_t* next_cache_len,
                                 const int32_t* out_tok, int32_t* grid_tok, int32_t* status,
                                 cudaStream_t stream);
// zero (nullable) [n_zero]: words cleared on the way (the fused lm_head's
// grid-barrier counters, lmhead_counters(), for a launch after this one).
cudaError_t launch_frontier(const ssd_grid& g, int32_t B, const int32_t* cache_len, int32_t D_max,
                            int32_t* n_drafts, int32_t* draft_pos, int32_t* status,
                            cudaStream_t stream, unsigned int* zero = nullptr,
                            int32_t n_zero = 0);
// pdl: launched as a programmatic dependent of the kernel before it on the
// stream (it may start while that kernel runs, needs none of its results and
// waits for it before exiting, so stream order is kept).
cudaError_t launch_counts(const ssd_grid& g, int32_t commit, int32_t B, int32_t D_max,
                          const int32_t* cache_len, const int32_t* n_drafts,
                          const uint8_t* accepted, int32_t* accepted_count,
                          int32_t* accepted_prefix, int32_t* next_cache_len, int32_t* status,
                          bool pdl, cudaStream_t stream);
// Commit pass: next cache length per sequence under SSD_COMMIT_NONE / BLOCK /
// FIRST_ROW of the frontier of cache_len under `g`.
cudaError_t launch_commit(const ssd_grid& g, int32_t commit, int32_t B, int32_t D_max,
                          const int32_t* cache_len, int32_t* next_cache_len, int32_t* status,
                          cudaStream_t stream);
// Staged schedule: slot j of every sequence takes slot W + j (j < W) of the
// per-row tokens and reference pointers.
cudaError_t launch_stage_shift(int32_t B, int32_t D_max, int32_t W, int32_t* tok,
                               const float** ref_rows, cudaStream_t stream);

// One warp: the counts of sequence b (a7) from its n drafts' accepted flags —
// drafts accepted, the leading accepted run and the next cache length under
// `commit` — written by lane 0 if `write`; every lane returns the leading run.  The
// drafts up to and including the first rejected one are committed (the
// rejected one with its resampled token); SSD_COMMIT_NONE / _BLOCK /
// _FIRST_ROW serve the verify-and-correct rounds, _PREFIX_BONUS the
// horizontal stage (Sec. 3.3, Sec. 4).
__device__ __forceinline__ int32_t sequence_counts(const ssd_grid& g, int32_t commit, int32_t b,
                                                   int32_t D_max, const int32_t* cache_len,
                                                   int32_t n, const uint8_t* accepted,
                                                   int32_t* accepted_count,
                                                   int32_t* accepted_prefix,
                                                   int32_t* next_cache_len, int32_t lane,
                                                   bool write = true) {
  int32_t count = 0, prefix = 0;
  bool run = true;  // still inside the leading accepted run
  for (int32_t j0 = 0; j0 < n; j0 += 32) {
    const int32_t j = j0 + lane;
    const bool a = (j < n) && accepted[(int64_t)b * D_max + j] != 0;
    const uint32_t acc_mask = __ballot_sync(0xffffffffu, a);
    count += __popc(acc_mask);
    if (run) {
      const uint32_t valid = (n - j0 >= 32) ? 0xffffffffu : ((1u << (n - j0)) - 1u);
      const uint32_t rejected = valid & ~acc_mask;
      if (rejected) {
        prefix += __ffs(rejected) - 1;
        run = false;
      } else {
        prefix += __popc(valid);
      }
    }
  }
  if (lane == 0 && write) {
    accepted_count[b] = count;
    accepted_prefix[b] = prefix;
    int32_t advance = n > 0 ? min(prefix + 1, n) : 0;  // SSD_COMMIT_PREFIX
    if (commit == SSD_COMMIT_NONE) {
      advance = 0;
    } else if (commit == SSD_COMMIT_BLOCK) {
      advance = n;
    } else if (commit == SSD_COMMIT_FIRST_ROW) {
      const int32_t n_c = cache_len[b] - g.prefix_len;
      advance = min(n, g.grid_w - n_c % g.grid_w);  // the frontier's first row
    } else if (commit == SSD_COMMIT_PREFIX_BONUS) {
      // horizontal stage: every draft accepted -> the bonus token as well, if
      // the position after the last draft exists (and has a row slot)
      const int32_t n_c = cache_len[b] - g.prefix_len;
      if (n > 0 && prefix == n && n < D_max && n_c + n < g.grid_h * g.grid_w) advance = n + 1;
    }
    next_cache_len[b] = cache_len[b] + advance;
  }
  return prefix;
}

// ---- accept.cu
struct AcceptArgs {
  int32_t rows, V;
  const float* tgt;
  const float* drf;
  int64_t ld;
  const int32_t* draft_tok;  // nullable
  float temperature;
  ssd_rng rng;
  int32_t* out_tok;
  uint8_t* accepted;
  float* ratio;              // nullable
  float* lse;                // nullable
  int32_t* status;
  const int32_t* n_drafts;   // nullable: row r valid iff r % D_max < n_drafts[r / D_max]
  int32_t D_max;
  int32_t strategy;          // ssd_strategy: (C) accept-reject, (A) greedy, (B) sampling
  const float** ref_rows;    // nullable: reference (draft) row of row r; a rejected row's entry
                             // is set to its target row (the next round's reference)
  int32_t ref_init;          // round 1: references are the draft rows; every entry is written
  int32_t bonus;             // horizontal stage: row j == n_drafts[b] draws the bonus token
  // Committed draws only (strategy (C) under the prefix rules, one round): the
  // kernel takes each row's decision in one pass, leaves out_tok = -1 on
  // rejected and bonus rows and writes the row's log2-domain normalisers
  // (Cp, Cq) to stats[r] (NaN: nothing to draw); launch_resolve then draws
  // the one token per sequence that the counts commit.
  int32_t lazy = 0;
  float2* stats = nullptr;   // [rows] when lazy
  // One verification step (rows = B * D_max): with cache_len non-null the
  // kernel computes every sequence's frontier under `grid` (Sec. 3.3) itself
  // instead of reading n_drafts, and spare lanes write it out (n_drafts_out,
  // draft_pos, as ssd_frontier) and zero `tickets` [B] for launch_resolve.
  const int32_t* cache_len = nullptr;
  ssd_grid grid{};
  int32_t* n_drafts_out = nullptr;
  int32_t* draft_pos = nullptr;
  int32_t* tickets = nullptr;
  // Under a programmatic launch of a kernel that reads none of this pass's
  // results (the step's attention): let it be scheduled at once, on the SMs
  // this pass leaves idle, instead of after the pass's last CTA.  0: never,
  // 1: always, 2: when the frontiers (cache_len non-null) hold at most one
  // row per two CTAs.
  int32_t early_dependents = 0;
};
bool accept_supported(int32_t V);
cudaError_t launch_accept(const AcceptArgs& a, cudaStream_t stream);
// After a lazy launch_accept on the same stream: per sequence b, the counts of
// sequence_counts() and the draw of the committed token — the residual token
// of the first rejected draft, or (bonus) the draw from p at the row after
// the last draft when every draft was accepted — bit-identical to the draw
// the eager kernel makes for that row.
struct ResolveArgs {
  ssd_grid grid;
  int32_t commit, B, D_max, V;
  const float* tgt;
  const float* drf;
  int64_t ld;
  float temperature;
  ssd_rng rng;
  const int32_t* cache_len;
  const int32_t* n_drafts;
  const float2* stats;
  int32_t bonus;
  int32_t* out_tok;
  uint8_t* accepted;
  int32_t* accepted_count;
  int32_t* accepted_prefix;
  int32_t* next_cache_len;
  int32_t* status;
  int32_t* tickets;  // [B], zeroed by the acceptance pass
  float* mass;       // [B][resolve_blocks(V)] block masses of the committed rows
};
int32_t resolve_blocks(int32_t V);
cudaError_t launch_resolve(const ResolveArgs& a, bool pdl, cudaStream_t stream);

// ---- attention.cu
struct AttnArgs {
  ssd_grid grid;
  int32_t B, Hq, Hkv, d, D_max, L_max;
  const int32_t* cache_len;
  const int32_t* n_drafts;
  const int32_t* draft_pos;
  const void* q;
  const void* k;
  const void* v;
  float scale;
  void* o;
  float* lse;  // nullable
  int32_t* status;
  // The step's frontier: the drafts of sequence b are its raster frontier under
  // `grid` (Sec. 3.3), computed from cache_len; n_drafts and draft_pos unread.
  int32_t raster = 0;
};
__device__ __forceinline__ int32_t attn_drafts(const AttnArgs& a, int32_t b) {
  if (!a.raster) return a.n_drafts[b];
  const int32_t n = frontier_drafts(a.grid, a.cache_len[b], a.D_max);
  return n < 0 ? 0 : n;  // an out-of-grid cache length is reported by the acceptance pass
}
// Grid index of draft j of sequence b.
__device__ __forceinline__ int32_t attn_draft_pos(const AttnArgs& a, int32_t b, int32_t j) {
  return a.raster ? a.cache_len[b] - a.grid.prefix_len + j
                  : a.draft_pos[(int64_t)b * a.D_max + j];
}
// Longest-first work order for the attention grids: CTA row `rank` (of B)
// takes the sequence with the rank-th most keys (cache_len + n_drafts, ties by
// index), so the longest sequences start in the first wave instead of being
// left for the last one.  A sequence with no drafts (a finished grid) has
// nothing to attend and ranks last, so its empty items do not take the first
// rounds of the dealing.  Batches above kLptMax keep their order.  Every
// thread of the block must call it; `skey` is shared memory of kLptMax + 1 ints.
constexpr int kLptMax = 256;
__device__ __forceinline__ int32_t longest_first(const AttnArgs& a, int32_t rank, int32_t* skey) {
  if (a.B > kLptMax) return rank;
  for (int32_t i = threadIdx.x; i < a.B; i += blockDim.x) {
    const int32_t c = a.cache_len[i], n = attn_drafts(a, i);
    skey[i] = (c >= 0 && n > 0 && c <= a.L_max && n <= a.D_max) ? c + n : 0;
  }
  __syncthreads();
  for (int32_t i = threadIdx.x; i < a.B; i += blockDim.x) {
    const int32_t k = skey[i];
    int32_t r = 0;
    for (int32_t j = 0; j < a.B; ++j) {
      const int32_t kj = skey[j];
      r += (kj > k) || (kj == k && j < i);
    }
    if (r == rank) skey[kLptMax] = i;  // the ranks form a permutation: one writer
  }
  __syncthreads();
  return skey[kLptMax];
}
size_t attention_workspace(int32_t B, int32_t Hq, int32_t Hkv, int32_t d, int32_t D_max,
                           int32_t L_max);
// defer_combine: leave the split-KV combine (if the plan has splits) to
// launch_attention_combine, so that another kernel can be queued between.
// pdl: the tcgen05 kernel is launched as a programmatic dependent of the kernel
// before it (it reads none of that kernel's results, starts as its CTAs retire,
// and lets the kernel after it be scheduled only once that kernel completed);
// the mma.sync kernel is always launched plainly.
cudaError_t launch_attention(const AttnArgs& a, void* ws, size_t ws_bytes, cudaStream_t stream,
                             bool defer_combine = false, bool pdl = false);
cudaError_t launch_attention_combine(const AttnArgs& a, void* ws, cudaStream_t stream);
int attention_launches(const ssd_grid& g, int32_t B, int32_t Hq, int32_t Hkv, int32_t d,
                       int32_t D_max, int32_t L_max);
// Most drafts one sequence can have under grid `g` (Sec. 3.3 frontier: at most
// min(k_h, W) horizontal positions, or W - c with k_h = 0, then k_v rows of W),
// clipped to D_max.
int32_t attention_rows_hint(const ssd_grid& g, int32_t D_max);

// ---- attention_tc.cu (tcgen05 frontier attention: query groups dividing 128,
// more than 64 query rows per KV group)
struct TcPlan {
  int32_t splits, kps, mtiles;
};
bool attention_tc_supported(int32_t Hq, int32_t Hkv, int32_t d, int32_t D_max);
TcPlan attention_tc_plan(int32_t B, int32_t Hq, int32_t Hkv, int32_t D_max, int32_t L_max);
cudaError_t launch_attention_tc(const AttnArgs& a, const TcPlan& p, int32_t* seq_ok, float* part_o,
                                float* part_lse, cudaStream_t stream, bool pdl = false);
// Same as launch_attention with the library's static device scratch as the
// workspace (ssd_verify_attention_noalloc); cudaErrorMemoryAllocation if the
// problem needs more than SSD_NOALLOC_SCRATCH_BYTES.
cudaError_t launch_attention_noalloc(const AttnArgs& a, cudaStream_t stream);

// ---- lmhead.cu
struct LmHeadArgs {
  int32_t rows, V, K;
  const void* h_tgt;
  const void* h_drf;
  const void* w_tgt;
  const void* w_drf;
  const int32_t* draft_tok;
  float temperature;
  ssd_rng rng;
  int32_t* out_tok;
  uint8_t* accepted;
  float* ratio;
  float* lse;
  int32_t* status;
  const int32_t* n_drafts;  // nullable, as AcceptArgs
  int32_t D_max;
  // With n_drafts: draw only the first rejected row of each sequence (the
  // token a one-round prefix commit keeps); other rejected rows get -1.
  int32_t lazy = 0;
  // The barrier words at the start of the workspace were cleared by a kernel
  // earlier on the stream (launch_frontier's `zero`): no memset.
  int32_t counters_zeroed = 0;
};
size_t lmhead_workspace(int32_t rows, int32_t V);
// The grid-barrier words at the start of a workspace and their count.
inline unsigned int* lmhead_counters(void* ws) { return static_cast<unsigned int*>(ws); }
constexpr int32_t kLmheadCounters = 2;
ssd_status lmhead_check(int32_t rows, int32_t V, int32_t K);
cudaError_t launch_lmhead(const LmHeadArgs& a, void* ws, size_t ws_bytes, cudaStream_t stream);

// ---- predictor.cu (Eq. 2: the spatial draft predictor and its draft tokens)
struct PredictorArgs {
  int32_t rows, d, m, V;
  const void* z;        // bf16 [rows][2d] = [h ; e]
  const void* w0;       // bf16 [d][2d]
  const void* w1;       // bf16 [m][d]
  const void* w3;       // bf16 [m][d]
  const void* w2;       // bf16 [d][m]
  const float* gamma1;  // [d]
  const float* gamma2;  // [d]
  const void* w_head;   // bf16 [d][V]
  float eps;
  int32_t* out_tok;     // [rows]
  float* out_hidden;    // fp32 [rows][d] or nullptr (then in the workspace)
};
// Workspace of launch_predictor (for the current device's SM count); 0 if
// the shape is unsupported.  More than 128 rows run as several launches, one
// per 128 rows, over the same workspace.
size_t predictor_workspace(int32_t rows, int32_t d, int32_t m, int32_t V, bool own_hidden);
bool predictor_supported(int32_t d, int32_t m, int32_t V);  // multiples of 128
cudaError_t launch_predictor(const PredictorArgs& p, void* ws, size_t ws_bytes, int32_t* status,
                             cudaStream_t stream);

int device_sm_count();

// cuTensorMapEncodeTiled, reached through the runtime's driver entry point
// (so the library loads without linking the driver); nullptr if unavailable.
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn tensor_map_encoder();
// A bf16 tensor map with the 128-byte swizzle: `rank` dimensions (innermost
// first), byte strides of dimensions 1.. and the box; false on failure.
bool bf16_tensor_map(CUtensorMap* map, const void* base, uint32_t rank, const uint64_t* dims,
                     const uint64_t* strides, const uint32_t* box);

// Failure-detection controls (ssd_set_wait_limit, ssd_set_barrier_shortfall),
// read by the host at every launch of a kernel with grid-wide waits: the poll
// limit of its bounded waits (kMaxPolls when unset) and the extra arrivals its
// grid barriers wait for (0 when unset; > 0 makes them run out).
uint32_t wait_poll_limit();
uint32_t barrier_shortfall();

}  // namespace ssd
