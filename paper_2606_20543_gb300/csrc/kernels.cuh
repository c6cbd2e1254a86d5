// kernels.cuh — internal launch interface between the C ABI (api.cu) and the
// kernels.  Not installed; callers use include/ssd.h.
#pragma once

#include "common.cuh"

namespace ssd {

// ---- frontier.cu
cudaError_t launch_frontier(const ssd_grid& g, int32_t B, const int32_t* cache_len, int32_t D_max,
                            int32_t* n_drafts, int32_t* draft_pos, int32_t* status,
                            cudaStream_t stream);
cudaError_t launch_counts(const ssd_grid& g, int32_t commit, int32_t B, int32_t D_max,
                          const int32_t* cache_len, const int32_t* n_drafts,
                          const uint8_t* accepted, int32_t* accepted_count,
                          int32_t* accepted_prefix, int32_t* next_cache_len, cudaStream_t stream);
// Staged schedule: slot j of every sequence takes slot W + j (j < W) of the
// per-row tokens and reference pointers.
cudaError_t launch_stage_shift(int32_t B, int32_t D_max, int32_t W, int32_t* tok,
                               const float** ref_rows, cudaStream_t stream);

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
};
bool accept_supported(int32_t V);
cudaError_t launch_accept(const AcceptArgs& a, cudaStream_t stream);

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
};
// Longest-first work order for the attention grids: CTA row `rank` (of B)
// takes the sequence with the rank-th most keys (cache_len + n_drafts, ties by
// index), so the longest sequences start in the first wave instead of being
// left for the last one.  Batches above kLptMax keep their order.  Every
// thread of the block must call it; `skey` is shared memory of kLptMax + 1 ints.
constexpr int kLptMax = 256;
__device__ __forceinline__ int32_t longest_first(const AttnArgs& a, int32_t rank, int32_t* skey) {
  if (a.B > kLptMax) return rank;
  for (int32_t i = threadIdx.x; i < a.B; i += blockDim.x) {
    const int32_t c = a.cache_len[i], n = a.n_drafts[i];
    skey[i] = (c >= 0 && n >= 0 && c <= a.L_max && n <= a.D_max) ? c + n : 0;
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
cudaError_t launch_attention(const AttnArgs& a, void* ws, size_t ws_bytes, cudaStream_t stream);
int attention_launches(int32_t B, int32_t Hq, int32_t Hkv, int32_t D_max, int32_t L_max);

// ---- attention_tc.cu (tcgen05 frontier attention: query groups dividing 128,
// more than 64 query rows per KV group)
struct TcPlan {
  int32_t splits, kps, mtiles;
};
bool attention_tc_supported(int32_t Hq, int32_t Hkv, int32_t d, int32_t D_max);
TcPlan attention_tc_plan(int32_t B, int32_t Hq, int32_t Hkv, int32_t D_max, int32_t L_max);
cudaError_t launch_attention_tc(const AttnArgs& a, const TcPlan& p, int32_t* seq_ok, float* part_o,
                                float* part_lse, cudaStream_t stream);
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
};
size_t lmhead_workspace(int32_t rows, int32_t V);
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
size_t predictor_workspace(int32_t rows, int32_t d, int32_t m, int32_t V, bool own_hidden);
cudaError_t launch_predictor(const PredictorArgs& p, void* ws, size_t ws_bytes,
                             cudaStream_t stream);

int device_sm_count();

}  // namespace ssd
