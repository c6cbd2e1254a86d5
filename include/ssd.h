/*
 * ssd.h — C ABI of libssd: the verification pass of Spatially Speculative
 * Decoding (SSD) on one GB300 (sm_103a).
 *
 * One verification step (Sec. 3.3, "Verification as Auto Correction") takes
 * the drafted frontier of every sequence (the remainder of the current grid
 * row, drafted by the horizontal heads, plus the row(s) directly below it,
 * drafted column-parallel by the vertical heads), scores it against the KV
 * cache under the spatial dependency mask, and accepts each draft with
 * probability min(p/q, 1) or replaces it by a draw from [p - q]_+.
 *
 * Conventions for every entry point:
 *  - Pointers marked "dev" are device pointers on the current CUDA device;
 *    "host" pointers are read during the call and not kept.  The caller owns
 *    every buffer; the library allocates nothing on these paths.  Workspace,
 *    where needed, is sized by the matching *_workspace() query and passed in.
 *  - All work is enqueued asynchronously on `stream` (NULL = the legacy
 *    default stream).  Nothing synchronises.
 *  - Host-side checks (null pointers, unsupported shapes, too little
 *    workspace) return a status synchronously and enqueue nothing.
 *    SSD_ERR_CUDA reports a failed launch (cudaGetLastError).
 *  - Device-side checks (a cache length outside [prefix, prefix + H*W], a
 *    draft position outside the grid, a draft token outside [0, V), a grid
 *    barrier that gave up waiting) record the FIRST error code in the device
 *    int32 `*status` with an atomic compare-and-swap from SSD_OK.  The library
 *    never clears `*status`; the caller zeroes it and reads it after a sync.
 *  - Row-major layouts, innermost index last.  bf16 buffers hold IEEE
 *    bfloat16 bit patterns (2 bytes per element).
 *  - Draft slot j of sequence b is row b*D_max + j of every per-draft array;
 *    slots j >= n_drafts[b] are padding: they are neither read nor used, and
 *    their per-row outputs are set to out_tok = -1, accepted = 0, ratio = 0.
 */
#ifndef SSD_H
#define SSD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t; declared here so callers need no CUDA header. */
typedef struct CUstream_st* ssd_stream_t;

typedef enum {
  SSD_OK = 0,
  SSD_ERR_INVALID_ARG = 1,   /* null pointer, negative size, bad enum       */
  SSD_ERR_SHAPE = 2,         /* sizes inconsistent with each other          */
  SSD_ERR_UNSUPPORTED = 3,   /* a valid shape this build has no kernel for  */
  SSD_ERR_CUDA = 4,          /* a CUDA call or launch failed                */
  SSD_ERR_TIMEOUT = 5,       /* device: a bounded grid-barrier wait expired */
  SSD_ERR_DEVICE_BOUNDS = 6, /* device: a position / token / length out of range */
  SSD_ERR_WORKSPACE = 7      /* workspace pointer null or too small         */
} ssd_status;

/* The image-token grid of Sec. 3.1 after its text prefix (Eq. 1).
 * Grid token (y, x) sits at flat sequence position
 *     prefix_len + y * row_stride + x.
 * row_stride is W, or W + 1 for backbones that close each row with an
 * end-of-line token.  k_v is the number of grid rows drafted below the
 * current one (vertical heads, Sec. 3.3); the frontier rule of
 * ssd_frontier() needs row_stride == W. */
typedef struct {
  int32_t grid_h;     /* H: grid rows                                     */
  int32_t grid_w;     /* W: grid columns                                  */
  int32_t row_stride; /* W or W + 1                                       */
  int32_t prefix_len; /* text-prefix tokens before grid token (0, 0)      */
  int32_t k_v;        /* rows drafted below the current row, >= 0 (0: the
                         rest of the current row only)                  */
  int32_t k_h;        /* horizontal drafts per step, >= 0 (0: the rest of
                         the row); with k_h < W - c the frontier is the
                         next k_h positions and no rows below            */
} ssd_grid;

/* Per-draft uniforms (u_acc, u_res).  If `uniforms` (dev, float32
 * [rows][2]) is non-NULL it is used as given.  Otherwise row r draws them
 * from Philox4x32-10 (Salmon et al., SC'11) with counter
 * (r, offset_lo, offset_hi, 0) and key (seed_lo, seed_hi):
 * u_acc = (x0 >> 8) * 2^-24, u_res = (x1 >> 8) * 2^-24. */
typedef struct {
  uint64_t seed;
  uint64_t offset;
  const float* uniforms;
} ssd_rng;

/* ABI version of this header (increment on any signature change). */
#define SSD_ABI_VERSION 9
int32_t ssd_abi_version(void);

/* Human-readable name of a status code (static string). */
const char* ssd_status_string(ssd_status s);

/* ---------------------------------------------------------------------------
 * Failure detection (no counterpart in the paper).  Every wait of a kernel on
 * another CTA, a copy or a product is bounded; a wait that runs out records
 * SSD_ERR_TIMEOUT in *status, and the kernel skips the rest of its work,
 * releases its tensor memory and returns, so the context stays usable.  Both
 * controls are process-wide and apply to launches enqueued after the call.
 *  ssd_set_wait_limit(polls): the polls after which each bounded wait of the
 *    kernels with grid-wide waits (the fused lm_head, the draft predictor)
 *    gives up; 0 restores the default, well above a second of waiting.
 *  ssd_set_barrier_shortfall(n): makes those kernels' grid-wide waits (the
 *    lm_head's grid barriers, the predictor's wait for the previous product)
 *    expect n arrivals more than their CTAs make, so that they cannot
 *    complete and run out after the wait limit: a way to exercise the timeout
 *    path without faulting anything.  0 (the default) turns it off.
 * ------------------------------------------------------------------------- */
void ssd_set_wait_limit(uint32_t max_polls);
void ssd_set_barrier_shortfall(uint32_t arrivals);

/* ---------------------------------------------------------------------------
 * a1. Frontier (Sec. 3.3: horizontal heads complete the current row, the
 * vertical heads draft the k_v rows below it; Sec. 3.1 raster order).
 * For each sequence b, with n_c = cache_len[b] - prefix_len committed grid
 * tokens and the first uncommitted token at (y0, c) = (n_c / W, n_c % W):
 *     n_drafts[b] = (W - c) + k_v * W, clipped at the grid's last row,
 *     or, with k_h > 0, h = min(k_h, W - c) horizontal drafts plus the k_v
 *     rows only when h = W - c (Sec. 3.3: k_h horizontal heads);
 *     draft_pos[b][j] = n_c + j (grid index y * W + x), j < n_drafts[b];
 * padding slots get -1.
 *   cache_len  dev int32 [B]
 *   n_drafts   dev int32 [B]             (out)
 *   draft_pos  dev int32 [B][D_max]      (out); D_max >= (k_v + 1) * W
 * Device errors: cache_len outside [prefix, prefix + H*W] -> DEVICE_BOUNDS
 * (that sequence gets n_drafts = 0).
 * ------------------------------------------------------------------------- */
ssd_status ssd_frontier(const ssd_grid* grid, int32_t B, const int32_t* cache_len,
                        int32_t D_max, int32_t* n_drafts, int32_t* draft_pos,
                        int32_t* status, ssd_stream_t stream);

/* ---------------------------------------------------------------------------
 * a2. Frontier attention (Sec. 3.3 "Verification as Auto Correction": the
 * drafted block passes through the backbone in parallel; App. "Deviation
 * from AR": each draft's context may hold other drafts).
 * For draft j of sequence b and query head h (KV head g = h / (Hq / Hkv)):
 *     O[b][j][h] = softmax_s(scale * Q[b][j][h] . K[b][g][s] + M(s, j)) V[b][g][s]
 * over key slots s < cache_len[b] + n_drafts[b].  Slots [0, cache_len) are
 * the committed cache (flat position s); slot cache_len + j' holds draft
 * j''s own key/value (flat position of draft_pos[b][j']).  M = 0 iff
 * pos(key) <= pos(query), else -inf.  scale = 0 selects 1/sqrt(d).
 *   q          dev bf16 [B][D_max][Hq][d]
 *   k, v       dev bf16 [B][Hkv][L_max][d]; cache_len + n_drafts <= L_max
 *   cache_len, n_drafts  dev int32 [B]
 *   draft_pos  dev int32 [B][D_max]  grid index y * W + x
 *   o          dev bf16 [B][D_max][Hq][d]   (out; padding slots untouched)
 *   lse        dev float32 [B][Hq][D_max] or NULL: log-sum-exp of the
 *              scaled scores (natural log)
 *   workspace  dev, >= ssd_verify_attention_workspace(...) bytes (split-KV
 *              partials and the schedule); may be NULL if that is 0.
 * Supported: d in {64, 128}; Hq % Hkv == 0; 1 <= D_max <= 128;
 * D_max * (Hq / Hkv) <= 512.  Device errors: a draft position outside the
 * grid or a key count above L_max -> DEVICE_BOUNDS (rows left untouched).
 * ------------------------------------------------------------------------- */
size_t ssd_verify_attention_workspace(int32_t B, int32_t Hq, int32_t Hkv, int32_t d,
                                      int32_t D_max, int32_t L_max);
ssd_status ssd_verify_attention(const ssd_grid* grid, int32_t B, int32_t Hq, int32_t Hkv,
                                int32_t d, const int32_t* cache_len, const int32_t* n_drafts,
                                const int32_t* draft_pos, int32_t D_max, int32_t L_max,
                                const void* q, const void* k, const void* v, float scale,
                                void* o, float* lse, void* workspace, size_t workspace_bytes,
                                int32_t* status, ssd_stream_t stream);

/* ---------------------------------------------------------------------------
 * Frontier attention without a caller-provided workspace.  The paper has no
 * counterpart: this is a deployment convenience of this library.
 * Some callers cannot allocate device memory at all, for example a plugin
 * inside an inference server whose host process has reserved all device
 * memory for its own pool, or a real-time decode loop that may not call
 * cudaMalloc because that call can synchronise the device and stall other
 * streams.  This entry point computes exactly what ssd_verify_attention()
 * computes (same arguments, minus the workspace), using instead a scratch
 * array of SSD_NOALLOC_SCRATCH_BYTES that the library holds in device memory
 * (a static __device__ array: every GPU that loads the library keeps it until
 * the process exits).  It allocates nothing and calls no allocating routine.
 *  - Limit: problems whose workspace (ssd_verify_attention_workspace()) is
 *    larger than SSD_NOALLOC_SCRATCH_BYTES are rejected with
 *    SSD_ERR_WORKSPACE before anything is enqueued.
 *  - Set-up: every call looks up the device address of the scratch array on
 *    the current device (cudaGetSymbolAddress).  The first call on a device
 *    is its set-up: it may load the library's device code there, so make it
 *    before any stream capture (and, after a device reset, make the next call
 *    outside a capture too).  Later look-ups are host-side only.  A failed
 *    look-up returns SSD_ERR_CUDA.
 *  - Sharing: every call on a device uses the same scratch array and leaves
 *    its contents behind.  Nothing in it needs to start at zero: each call
 *    writes every scratch word it later reads.  Calls that overlap on the
 *    GPU (other streams, other host threads) race on the array and must be
 *    serialised by the caller.
 * ------------------------------------------------------------------------- */
#define SSD_NOALLOC_SCRATCH_BYTES ((size_t)64 << 20)
ssd_status ssd_verify_attention_noalloc(const ssd_grid* grid, int32_t B, int32_t Hq, int32_t Hkv,
                                        int32_t d, const int32_t* cache_len,
                                        const int32_t* n_drafts, const int32_t* draft_pos,
                                        int32_t D_max, int32_t L_max, const void* q, const void* k,
                                        const void* v, float scale, void* o, float* lse,
                                        int32_t* status, ssd_stream_t stream);

/* ---------------------------------------------------------------------------
 * a3-a5. Acceptance (Sec. 3.3 strategy (C); temperature of App.
 * "Configuration").  For every row r < rows:
 *     p = softmax(tgt[r] / T), q = softmax(drf[r] / T)
 *     t = draft_tok[r], or argmax_v drf[r][v] (lowest index on ties) if NULL
 *     ratio = p(t) / q(t) (evaluated in log space)
 *     accept iff u_acc < min(ratio, 1)
 *     on reject: out = smallest v with sum_{v' <= v} [p - q]_+ > u_res * Z,
 *                Z = sum_v [p - q]_+ (if Z == 0: the same draw from p)
 *   tgt_logits, drf_logits  dev float32, row r at + r * ld, V entries;
 *                           16-byte aligned, ld % 4 == 0, V % 4 == 0
 *   draft_tok  dev int32 [rows] or NULL
 *   out_tok    dev int32 [rows] (out); accepted dev uint8 [rows] (out)
 *   ratio      dev float32 [rows] or NULL (out)
 *   lse        dev float32 [rows][2] or NULL (out): log-sum-exp of tgt/T and
 *              of drf/T
 * Device errors: draft_tok outside [0, V) -> DEVICE_BOUNDS (row gets
 * out_tok = -1, accepted = 0).
 * ------------------------------------------------------------------------- */
ssd_status ssd_accept(int32_t rows, int32_t V, const float* tgt_logits, const float* drf_logits,
                      int64_t ld, const int32_t* draft_tok, float temperature, const ssd_rng* rng,
                      int32_t* out_tok, uint8_t* accepted, float* ratio, float* lse,
                      int32_t* status, ssd_stream_t stream);

/* ---------------------------------------------------------------------------
 * The three token-selection strategies of Sec. 3.3, applied to every row
 * independently with the p, q, t, ratio and lse of ssd_accept():
 *   SSD_STRATEGY_ACCEPT_REJECT  (C) the rule of ssd_accept() (the default)
 *   SSD_STRATEGY_GREEDY         (A) out = argmax_v tgt[r][v] (lowest index
 *                               on ties); accepted = (out == t)
 *   SSD_STRATEGY_SAMPLE         (B) out = smallest v with
 *                               sum_{v' <= v} p(v') > u_res * sum_v p(v);
 *                               accepted = (out == t)
 * ratio and lse are filled as by ssd_accept() under every strategy.
 * An unknown strategy returns SSD_ERR_INVALID_ARG before any launch.
 * ------------------------------------------------------------------------- */
typedef enum {
  SSD_STRATEGY_ACCEPT_REJECT = 0,
  SSD_STRATEGY_GREEDY = 1,
  SSD_STRATEGY_SAMPLE = 2
} ssd_strategy;
ssd_status ssd_accept_strategy(int32_t strategy, int32_t rows, int32_t V, const float* tgt_logits,
                               const float* drf_logits, int64_t ld, const int32_t* draft_tok,
                               float temperature, const ssd_rng* rng, int32_t* out_tok,
                               uint8_t* accepted, float* ratio, float* lse, int32_t* status,
                               ssd_stream_t stream);

/* ---------------------------------------------------------------------------
 * One verify-and-correct round (Sec. 3.3: the verify-and-correct procedure
 * runs for a fixed number r of rounds; a position rejected in one round takes
 * that round's backbone distribution as its reference in the next, and an
 * accepted position keeps the reference it has).
 * For every row r the rule of ssd_accept_strategy() is applied with
 *     q = softmax(ref_rows[r][0 .. V) / T)   (the row's current reference)
 *     t = tok[r]                             (the position's current token;
 *                                             NULL: argmax of the reference row,
 *                                             the draft token of round 1)
 * and, when the row is not accepted, ref_rows[r] is set to tgt + r * ld, so
 * this round's distribution is the row's reference in the next round.  Round
 * 1 passes pointers to the draft rows and the draft tokens; out_tok is the
 * next round's tok.  Give every round its own rng offset.
 *   ref_rows  dev [rows] of const float* (in/out), each 16-byte aligned
 *   tok       dev int32 [rows] or NULL
 *   other arguments as ssd_accept_strategy().
 * ------------------------------------------------------------------------- */
ssd_status ssd_accept_round(int32_t strategy, int32_t rows, int32_t V, const float* tgt_logits,
                            int64_t ld, const float** ref_rows, const int32_t* tok,
                            float temperature, const ssd_rng* rng, int32_t* out_tok,
                            uint8_t* accepted, float* ratio, float* lse, int32_t* status,
                            ssd_stream_t stream);

/* Commit rule of the counts of ssd_verify_step() (a7):
 *   SSD_COMMIT_PREFIX     one round: the drafts up to and including the first
 *                         rejected one (the horizontal stage; the default)
 *   SSD_COMMIT_NONE       a round before the last: nothing is committed
 *   SSD_COMMIT_BLOCK      the last of r rounds: the whole corrected block
 *   SSD_COMMIT_FIRST_ROW  the staged schedule's first commit: the frontier's
 *                         first row, W - (cache_len - prefix_len) % W drafts
 *   SSD_COMMIT_PREFIX_BONUS the horizontal stage (Sec. 4: one round): the
 *                         prefix rule, and when every draft is accepted the
 *                         bonus token as well, so next = cache + n_d + 1 if
 *                         the position after the last draft exists.  Row
 *                         b * D_max + n_d of the target logits then holds the
 *                         backbone's logits at that position (n_d < D_max);
 *                         its out_tok is the bonus token: under (A) the argmax
 *                         of p, otherwise a draw from p with the row's u_res;
 *                         its accepted flag is 1.  Logits path only. */
typedef enum {
  SSD_COMMIT_PREFIX = 0,
  SSD_COMMIT_NONE = 1,
  SSD_COMMIT_BLOCK = 2,
  SSD_COMMIT_FIRST_ROW = 3,
  SSD_COMMIT_PREFIX_BONUS = 4
} ssd_commit;

/* Commit pass (Sec. 3.3: after the final round one more forward pass commits
 * the corrected block and updates the KV cache).  For every sequence b, with
 * the frontier of cache_len[b] under `grid` (as ssd_frontier):
 *   SSD_COMMIT_BLOCK      next_cache_len[b] = cache_len[b] + n_drafts
 *   SSD_COMMIT_FIRST_ROW  next_cache_len[b] = cache_len[b] + min(n_drafts, W - c)
 *   SSD_COMMIT_NONE       next_cache_len[b] = cache_len[b]
 * The pass's attention over the committed block is ssd_verify_attention; the
 * committed tokens are the ones the last round left (the pass changes none).
 * The prefix rules need accept decisions (ssd_verify_step): they return
 * SSD_ERR_INVALID_ARG.  Device errors: cache_len outside the grid ->
 * DEVICE_BOUNDS (next_cache_len = cache_len).
 *   cache_len, next_cache_len  dev int32 [B] (may alias) */
ssd_status ssd_commit_pass(const ssd_grid* grid, int32_t B, const int32_t* cache_len,
                           int32_t D_max, int32_t commit, int32_t* next_cache_len,
                           int32_t* status, ssd_stream_t stream);

/* Staged schedule (App. multi-row, "commit the first row, then refine the
 * trailing row"): for every sequence b and j < W, slot b * D_max + j of tok
 * and of ref_rows (may be NULL) takes slot b * D_max + W + j, so the
 * trailing row of a two-row frontier becomes the frontier of the incremental
 * rounds (k_v = 0).  Requires 2 * W <= D_max. */
ssd_status ssd_stage_shift(int32_t B, int32_t D_max, int32_t W, int32_t* tok,
                           const float** ref_rows, ssd_stream_t stream);

/* The tokens one step committed, into each sequence's grid (Sec. 3.3: the
 * accepted prefix, then the first rejected draft's resampled token, fill the
 * next raster positions).  For every b, with n_c = cache_len[b] - prefix_len
 * and adv = next_cache_len[b] - cache_len[b]:
 *     grid_tok[b][n_c + j] = out_tok[b * D_max + j],  0 <= j < adv.
 * Call it after a step and before next_cache_len becomes cache_len; with it
 * the grid, the cache lengths and the step index are the whole state of a
 * replay (paper_2606_20543_gb300.step.ReplayState dumps and restores them).
 *   cache_len, next_cache_len  dev int32 [B];  out_tok dev int32 [B * D_max]
 *   grid_tok   dev int32 [B][hw] (in/out: only the committed slots change)
 * A sequence whose advance leaves [0, D_max] or the grid records
 * SSD_ERR_DEVICE_BOUNDS in *status and writes nothing. */
ssd_status ssd_record_commit(int32_t B, int32_t D_max, int32_t prefix_len, int32_t hw,
                             const int32_t* cache_len, const int32_t* next_cache_len,
                             const int32_t* out_tok, int32_t* grid_tok, int32_t* status,
                             ssd_stream_t stream);

/* ---------------------------------------------------------------------------
 * a6. Fused lm_head + acceptance (Sec. 3.3, after Eq. 2: tokens are decoded
 * through the base model's GenHead).  Logits l_p = H_t W_t and l_q = H_d W_d
 * are formed on chip (tcgen05, fp32 accumulation) and fed to the rule of
 * ssd_accept() without being written to memory.
 *   h_tgt, h_drf  dev bf16 [rows][K] (already normalised hidden states)
 *   w_tgt, w_drf  dev bf16 [K][V]   (may alias each other)
 *   other arguments as ssd_accept(); lse may be NULL.
 *   workspace     dev, >= ssd_lmhead_accept_workspace(rows, V) bytes
 * Supported: 1 <= rows <= 256, K % 64 == 0, V % 128 == 0, V / 128 no more
 * than the co-resident CTAs of the device.  The kernel's CTAs meet at three
 * bounded grid barriers; a barrier that waits too long records
 * SSD_ERR_TIMEOUT and the kernel returns without writing its outputs (the
 * first barrier; a later one leaves the decisions written before it).
 * ------------------------------------------------------------------------- */
size_t ssd_lmhead_accept_workspace(int32_t rows, int32_t V);
ssd_status ssd_lmhead_accept(int32_t rows, int32_t V, int32_t K, const void* h_tgt,
                             const void* h_drf, const void* w_tgt, const void* w_drf,
                             const int32_t* draft_tok, float temperature, const ssd_rng* rng,
                             int32_t* out_tok, uint8_t* accepted, float* ratio, float* lse,
                             void* workspace, size_t workspace_bytes, int32_t* status,
                             ssd_stream_t stream);

/* ---------------------------------------------------------------------------
 * a1-a7. One whole verification step: frontier (a1), frontier attention
 * (a2), acceptance from logits (a3-a5) or from hidden states through the
 * fused lm_head (a6), and the counts that advance the cache (a7):
 *     accepted_count[b]  = drafts of b accepted
 *     accepted_prefix[b] = leading drafts of b (raster order) accepted
 *     next_cache_len[b]  = cache_len[b] + min(accepted_prefix[b] + 1, n_d)
 *                          (the first rejected draft carries its resampled
 *                          token; an empty frontier leaves cache_len as is)
 * Acceptance rows are b*D_max + j; the Philox counter row is the same index.
 * Logits path: tgt_logits/drf_logits non-NULL ([B*D_max] rows of ld floats).
 * Fused path:  logits NULL and h_tgt, h_drf, w_tgt, w_drf non-NULL (hidden
 *              = K of ssd_lmhead_accept).
 * strategy: an ssd_strategy for the logits path; the fused path supports
 * SSD_STRATEGY_ACCEPT_REJECT only (others: SSD_ERR_UNSUPPORTED).
 * ref_rows: NULL, or the per-row references of a verify-and-correct round
 * (see ssd_accept_round(); logits path only).  ref_init = 1 marks round 1:
 * the references are the draft rows (drf_logits) and every entry of
 * ref_rows is written (the draft row, or the target row when the row is
 * not accepted), so no pass over ref_rows is needed before a block.
 * commit: an ssd_commit; the counts' next_cache_len follows it.
 * out->next_cache_len must not overlap args->cache_len (SSD_ERR_INVALID_ARG):
 * the counts run beside the attention, which reads cache_len.
 * ssd_verify_accept() runs its kernels in stream order and allows it.
 * Draws: under strategy (C) from logits with commit SSD_COMMIT_PREFIX or
 * SSD_COMMIT_PREFIX_BONUS and no ref_rows, the step draws only the token it
 * commits: the residual token of each sequence's first rejected draft, or
 * the bonus token when every draft is accepted.  out_tok of the other
 * rejected rows (never committed: the drafts after the first rejection are
 * discarded) and of an uncommitted bonus row is -1; accepted and ratio are
 * written for every row.  The committed token is the one the full draw
 * (ssd_accept_strategy) gives for that row, bit for bit.  The fused path
 * with SSD_COMMIT_PREFIX draws likewise only each sequence's first rejected
 * draft.  The other commit rules, ref_rows and strategies (A) and (B) draw
 * every row.
 * Streams: logits path — the acceptance pass computes the frontier itself
 * (and writes n_drafts and draft_pos) and the attention computes the same
 * frontier from cache_len.  With at least 2 x (SM count) rows and either
 * committed draws only, or strategy (A) with at most (SM count) rows that can
 * hold a draft, everything runs on `stream`: acceptance, attention,
 * then the counts (and committed draws) as a programmatic dependent of the
 * attention (they need only the acceptance's results, start once every
 * attention CTA is resident and wait for the attention before they exit, so
 * stream order holds).  Otherwise, and on the fused path (frontier first,
 * lm_head acceptance), the acceptance and counts run on a side stream beside
 * the attention, joined back into `stream`; the library creates that stream
 * once per device and host thread (with two events).  Make the first call on
 * each device and host thread outside any stream capture; later calls may
 * be captured (the fork and join become graph edges).
 * ------------------------------------------------------------------------- */
typedef struct {
  ssd_grid grid;
  int32_t B, Hq, Hkv, d, D_max, L_max, V;
  const int32_t* cache_len;   /* dev int32 [B]                         */
  const void* q;              /* dev bf16 [B][D_max][Hq][d]            */
  const void* k;              /* dev bf16 [B][Hkv][L_max][d]           */
  const void* v;              /* dev bf16 [B][Hkv][L_max][d]           */
  float scale;                /* 0 -> 1/sqrt(d)                        */
  const float* tgt_logits;    /* dev float32 [B*D_max][ld] or NULL     */
  const float* drf_logits;    /* dev float32 [B*D_max][ld] or NULL     */
  int64_t ld;
  const void* h_tgt;          /* dev bf16 [B*D_max][hidden] or NULL    */
  const void* h_drf;
  const void* w_tgt;          /* dev bf16 [hidden][V] or NULL          */
  const void* w_drf;
  int32_t hidden;
  const int32_t* draft_tok;   /* dev int32 [B*D_max] or NULL (argmax q)*/
  float temperature;
  ssd_rng rng;
  int32_t strategy;           /* ssd_strategy (0: accept-reject)       */
  const float** ref_rows;     /* dev [B*D_max] or NULL (round refs)    */
  int32_t ref_init;           /* 1: round 1 (writes every ref_rows)    */
  int32_t commit;             /* ssd_commit (0: prefix rule)           */
} ssd_verify_args;

typedef struct {
  int32_t* n_drafts;          /* dev int32 [B]                          */
  int32_t* draft_pos;         /* dev int32 [B][D_max]                   */
  void* o;                    /* dev bf16 [B][D_max][Hq][d]             */
  float* lse;                 /* dev float32 [B][Hq][D_max] or NULL     */
  int32_t* out_tok;           /* dev int32 [B*D_max]                    */
  uint8_t* accepted;          /* dev uint8 [B*D_max]                    */
  float* ratio;               /* dev float32 [B*D_max] or NULL          */
  int32_t* accepted_count;    /* dev int32 [B]                          */
  int32_t* accepted_prefix;   /* dev int32 [B]                          */
  int32_t* next_cache_len;    /* dev int32 [B]                          */
  int32_t* status;            /* dev int32 [1]                          */
} ssd_verify_out;

size_t ssd_verify_step_workspace(const ssd_verify_args* args);
/* Number of kernels one ssd_verify_step() with these arguments launches
 * (host query, no GPU work); -1 if the arguments would be rejected. */
int32_t ssd_verify_step_launches(const ssd_verify_args* args);
ssd_status ssd_verify_step(const ssd_verify_args* args, const ssd_verify_out* out,
                           void* workspace, size_t workspace_bytes, ssd_stream_t stream);

/* ssd_verify_step() without the attention (a1, a3-a5, a7), on `stream`
 * alone: the frontier (written to out->n_drafts and out->draft_pos), the
 * acceptance with its committed draws, and the counts.  Uses args->grid, B,
 * D_max, V, cache_len, the logits (or hidden-state) fields, draft_tok,
 * temperature, rng, strategy, ref_rows, ref_init and commit; Hq, Hkv, d,
 * L_max, q, k, v, scale and out->o, out->lse are ignored.  workspace:
 * ssd_verify_step_workspace(args) bytes are enough.  Errors as
 * ssd_verify_step(). */
ssd_status ssd_verify_accept(const ssd_verify_args* args, const ssd_verify_out* out,
                             void* workspace, size_t workspace_bytes, ssd_stream_t stream);

/* ---------------------------------------------------------------------------
 * The spatial draft predictor (Sec. 3.3 "Draft Prediction in Latent Space",
 * Eq. 2) and its draft tokens, for `rows` positions at once (one grid row of
 * W columns for a vertical head, or the k_h horizontal offsets):
 *     h_hat = W0 z + W2 (silu(W1 a) * W3 a),  a = RMSNorm(W0 z; gamma1),
 *     out_tok = argmax_v (RMSNorm(h_hat; gamma2) W_head)_v  (lowest index on
 *     ties), RMSNorm(x; g) = x / sqrt(mean(x^2) + eps) * g.
 *   z        dev bf16 [rows][2d]: [h ; e], the hidden state and the token
 *            embedding of each source position
 *   w0       dev bf16 [d][2d]; w1, w3 dev bf16 [m][d]; w2 dev bf16 [d][m]
 *            ([out][in], as a linear layer stores them)
 *   gamma1, gamma2  dev float32 [d]; w_head dev bf16 [d][V] (GenHead)
 *   out_tok  dev int32 [rows] (out); out_hidden dev float32 [rows][d] or NULL
 *            (out: h_hat, the predicted pre-norm hidden state)
 *   workspace dev, >= ssd_draft_predict_workspace(rows, d, m, V) bytes
 * Every product input is bf16 with fp32 accumulation on the tensor cores
 * (one cooperative kernel, one CTA per SM, streams every weight matrix once;
 * more than 128 rows run as one launch per 128 rows).  The workspace size
 * depends on the current device's SM count.  The kernel's CTAs wait on each
 * other between the products with bounded waits: one that runs out records
 * SSD_ERR_TIMEOUT and the call writes no tokens.
 * Supported: rows >= 1; d, m and V multiples of 128 (other multiples of 8 /
 * 4 return SSD_ERR_UNSUPPORTED); every pointer 16-byte aligned.
 * ------------------------------------------------------------------------- */
size_t ssd_draft_predict_workspace(int32_t rows, int32_t d, int32_t m, int32_t V);
ssd_status ssd_draft_predict(int32_t rows, int32_t d, int32_t m, int32_t V, const void* z,
                             const void* w0, const void* w1, const void* w3, const void* w2,
                             const float* gamma1, const float* gamma2, const void* w_head,
                             float eps, int32_t* out_tok, float* out_hidden, void* workspace,
                             size_t workspace_bytes, int32_t* status, ssd_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* SSD_H */
