// frontier.cu — the drafted frontier (step a1) and the accepted counts /
// next cache length (step a7) of one verification step.
//
// Frontier (Sec. 3.3): the horizontal heads complete the current grid row,
// the vertical heads draft the k_v rows below it in one column-parallel step.
// With n_c committed grid tokens and the first uncommitted one at
// (y0, c) = (n_c / W, n_c % W), the frontier is the next
// (W - c) + k_v * W raster positions, clipped at the last grid row.  With
// k_h > 0 the horizontal part is the next min(k_h, W - c) positions (k_h
// horizontal heads), and the vertical rows follow only when it completes
// the row, so the frontier stays one contiguous raster run.
//
// Counts (Sec. 3.3 and Sec. 4 "SSD Configuration", one verification round):
// the drafts up to and including the first rejected one are committed, the
// rejected one carrying its resampled token.  With r verify-and-correct
// rounds (Sec. 3.3) the rounds before the last commit nothing and the last
// commits the whole corrected block; the staged schedule (App. multi-row)
// commits the frontier's first row after its base rounds.  The horizontal
// stage (Sec. 4, one round) adds the bonus token when every draft is kept.
#include "kernels.cuh"

namespace ssd {

// One block per sequence.  Writes n_drafts[b] and draft_pos[b][0..D_max);
// block 0 also clears `zero` [n_zero] (the grid-barrier words of the kernel
// that follows, which then needs no memset of its own).
__global__ void frontier_kernel(ssd_grid g, const int32_t* __restrict__ cache_len, int32_t D_max,
                                int32_t* __restrict__ n_drafts, int32_t* __restrict__ draft_pos,
                                int32_t* status, unsigned int* zero, int32_t n_zero) {
  const int32_t b = blockIdx.x;
  if (b == 0)
    for (int32_t i = threadIdx.x; i < n_zero; i += blockDim.x) zero[i] = 0u;
  const int32_t n_c = cache_len[b] - g.prefix_len;
  const int32_t n = frontier_drafts(g, cache_len[b], D_max);
  if (threadIdx.x == 0) {
    n_drafts[b] = n < 0 ? 0 : n;
    if (n < 0) record_status(status, SSD_ERR_DEVICE_BOUNDS);
  }
  for (int32_t j = threadIdx.x; j < D_max; j += blockDim.x)
    draft_pos[(int64_t)b * D_max + j] = (j < n) ? (n_c + j) : -1;
}

// One warp per sequence: accepted count, leading accepted run, next length.
__global__ void counts_kernel(ssd_grid g, int32_t commit, int32_t B, int32_t D_max,
                              const int32_t* __restrict__ cache_len,
                              const int32_t* __restrict__ n_drafts,
                              const uint8_t* __restrict__ accepted,
                              int32_t* __restrict__ accepted_count,
                              int32_t* __restrict__ accepted_prefix,
                              int32_t* __restrict__ next_cache_len, int32_t* status) {
  const int32_t b = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (b >= B) {
    if (pdl_first_block()) pdl_wait();
    return;
  }
  int32_t n = n_drafts[b];
  if (n < 0 || n > D_max) {  // a caller's frontier (ssd_verify_accept) out of range
    if ((threadIdx.x & 31) == 0) record_status(status, SSD_ERR_DEVICE_BOUNDS);
    n = n < 0 ? 0 : D_max;
  }
  sequence_counts(g, commit, b, D_max, cache_len, n, accepted, accepted_count, accepted_prefix,
                  next_cache_len, threadIdx.x & 31);
  // under a programmatic launch: block 0 exits only after the kernel before it
  if (pdl_first_block()) pdl_wait();
}

// Staged schedule: the trailing row (slots W .. 2W-1) becomes the frontier of
// the incremental rounds (slots 0 .. W-1), with its tokens and references.
__global__ void stage_shift_kernel(int32_t B, int32_t D_max, int32_t W, int32_t* __restrict__ tok,
                                   const float** __restrict__ ref_rows) {
  const int32_t b = blockIdx.x;
  for (int32_t j = threadIdx.x; j < W; j += blockDim.x) {
    const int64_t dst = (int64_t)b * D_max + j, src = dst + W;
    // destination slots 0 .. W-1 and source slots W .. 2W-1 do not overlap
    const int32_t t = tok[src];
    const float* p = ref_rows != nullptr ? ref_rows[src] : nullptr;
    tok[dst] = t;
    if (ref_rows != nullptr) ref_rows[dst] = p;
  }
}

// Commit pass (Sec. 3.3: after the final round one more forward pass commits
// the corrected block): the next cache length of every sequence under a
// commit rule that needs no accept decisions.
__global__ void commit_kernel(ssd_grid g, int32_t commit, int32_t B, int32_t D_max,
                              const int32_t* __restrict__ cache_len,
                              int32_t* __restrict__ next_cache_len, int32_t* status) {
  const int32_t b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  const int32_t cl = cache_len[b];
  const int32_t n = frontier_drafts(g, cl, D_max);
  if (n < 0) {
    record_status(status, SSD_ERR_DEVICE_BOUNDS);
    next_cache_len[b] = cl;
    return;
  }
  int32_t advance = 0;
  if (commit == SSD_COMMIT_BLOCK) {
    advance = n;
  } else if (commit == SSD_COMMIT_FIRST_ROW) {
    const int32_t n_c = cl - g.prefix_len;
    advance = min(n, g.grid_w - n_c % g.grid_w);
  }
  next_cache_len[b] = cl + advance;
}

cudaError_t launch_commit(const ssd_grid& g, int32_t commit, int32_t B, int32_t D_max,
                          const int32_t* cache_len, int32_t* next_cache_len, int32_t* status,
                          cudaStream_t stream) {
  if (B == 0) return cudaSuccess;
  commit_kernel<<<(B + 127) / 128, 128, 0, stream>>>(g, commit, B, D_max, cache_len,
                                                     next_cache_len, status);
  return cudaGetLastError();
}

// The committed tokens of one step into each sequence's grid (Sec. 3.3: the
// accepted prefix and the first rejected draft's resampled token take the
// next raster positions).  One block per sequence: the step advanced the cache
// from cache_len[b] to next_cache_len[b], i.e. tokens out_tok[b][0 .. adv) at
// grid positions n_c .. n_c + adv.
__global__ void record_commit_kernel(int32_t D_max, int32_t prefix_len, int32_t hw,
                                     const int32_t* __restrict__ cache_len,
                                     const int32_t* __restrict__ next_cache_len,
                                     const int32_t* __restrict__ out_tok,
                                     int32_t* __restrict__ grid_tok, int32_t* status) {
  const int32_t b = blockIdx.x;
  const int32_t n_c = cache_len[b] - prefix_len;
  const int32_t adv = next_cache_len[b] - cache_len[b];
  if (n_c < 0 || adv < 0 || adv > D_max || n_c + adv > hw) {
    if (threadIdx.x == 0) record_status(status, SSD_ERR_DEVICE_BOUNDS);
    return;
  }
  for (int32_t j = threadIdx.x; j < adv; j += blockDim.x)
    grid_tok[(int64_t)b * hw + n_c + j] = out_tok[(int64_t)b * D_max + j];
}

cudaError_t launch_record_commit(int32_t B, int32_t D_max, int32_t prefix_len, int32_t hw,
                                 const int32_t* cache_len, const int32_t* next_cache_len,
                                 const int32_t* out_tok, int32_t* grid_tok, int32_t* status,
                                 cudaStream_t stream) {
  if (B == 0) return cudaSuccess;
  record_commit_kernel<<<B, 128, 0, stream>>>(D_max, prefix_len, hw, cache_len, next_cache_len,
                                              out_tok, grid_tok, status);
  return cudaGetLastError();
}

cudaError_t launch_frontier(const ssd_grid& g, int32_t B, const int32_t* cache_len, int32_t D_max,
                            int32_t* n_drafts, int32_t* draft_pos, int32_t* status,
                            cudaStream_t stream, unsigned int* zero, int32_t n_zero) {
  if (B == 0) return cudaSuccess;
  frontier_kernel<<<B, 128, 0, stream>>>(g, cache_len, D_max, n_drafts, draft_pos, status, zero,
                                         zero != nullptr ? n_zero : 0);
  return cudaGetLastError();
}

cudaError_t launch_counts(const ssd_grid& g, int32_t commit, int32_t B, int32_t D_max,
                          const int32_t* cache_len, const int32_t* n_drafts,
                          const uint8_t* accepted, int32_t* accepted_count,
                          int32_t* accepted_prefix, int32_t* next_cache_len, int32_t* status,
                          bool pdl, cudaStream_t stream) {
  if (B == 0) return cudaSuccess;
  const int warps = 4;
  return launch_kernel(counts_kernel, dim3((B + warps - 1) / warps), dim3(warps * 32), 0, stream,
                       pdl, g, commit, B, D_max, cache_len, n_drafts, accepted, accepted_count,
                       accepted_prefix, next_cache_len, status);
}

cudaError_t launch_stage_shift(int32_t B, int32_t D_max, int32_t W, int32_t* tok,
                               const float** ref_rows, cudaStream_t stream) {
  if (B == 0 || W == 0) return cudaSuccess;
  stage_shift_kernel<<<B, 128, 0, stream>>>(B, D_max, W, tok, ref_rows);
  return cudaGetLastError();
}

}  // namespace ssd
