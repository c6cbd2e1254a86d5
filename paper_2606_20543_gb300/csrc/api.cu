// api.cu — the extern "C" entry points of libssd declared in include/ssd.h:
// host-side argument checks, workspace carving, and kernel launches on the
// caller's stream.  No allocation, no synchronisation.
#include <math.h>

#include <algorithm>
#include <atomic>

#include "kernels.cuh"

using namespace ssd;

namespace ssd {

namespace {
std::atomic<uint32_t> g_wait_polls{0};
std::atomic<uint32_t> g_barrier_shortfall{0};
}  // namespace

uint32_t wait_poll_limit() {
  const uint32_t p = g_wait_polls.load(std::memory_order_relaxed);
  return p == 0 ? kMaxPolls : p;
}
uint32_t barrier_shortfall() { return g_barrier_shortfall.load(std::memory_order_relaxed); }

}  // namespace ssd

namespace {

ssd_status from_cuda(cudaError_t e) { return e == cudaSuccess ? SSD_OK : SSD_ERR_CUDA; }

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Side stream of ssd_verify_step: acceptance runs on it, concurrently with the
// attention of the same step on the caller's stream (they share no data).
// One per device and host thread, created on first use and kept until exit.
struct SideStream {
  cudaStream_t stream = nullptr;
  cudaEvent_t fork = nullptr, join = nullptr;
};
constexpr int kMaxSideDevices = 64;

cudaError_t side_stream(SideStream** out) {
  thread_local SideStream side[kMaxSideDevices];
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxSideDevices) return cudaErrorInvalidDevice;
  SideStream& s = side[dev];
  if (s.stream == nullptr) {
    if ((e = cudaStreamCreateWithFlags(&s.stream, cudaStreamNonBlocking)) != cudaSuccess) return e;
    if ((e = cudaEventCreateWithFlags(&s.fork, cudaEventDisableTiming)) != cudaSuccess) return e;
    if ((e = cudaEventCreateWithFlags(&s.join, cudaEventDisableTiming)) != cudaSuccess) return e;
  }
  *out = &s;
  return cudaSuccess;
}

ssd_status check_grid(const ssd_grid* g) {
  if (g == nullptr) return SSD_ERR_INVALID_ARG;
  if (g->grid_h <= 0 || g->grid_w <= 0 || g->prefix_len < 0 || g->k_v < 0 || g->k_h < 0)
    return SSD_ERR_SHAPE;
  if (g->row_stride != g->grid_w && g->row_stride != g->grid_w + 1) return SSD_ERR_SHAPE;
  if ((int64_t)g->grid_h * g->row_stride + g->prefix_len > INT32_MAX / 2) return SSD_ERR_SHAPE;
  return SSD_OK;
}

ssd_status check_attention(const ssd_grid* grid, int32_t B, int32_t Hq, int32_t Hkv, int32_t d,
                           int32_t D_max, int32_t L_max) {
  ssd_status s = check_grid(grid);
  if (s != SSD_OK) return s;
  if (B < 0 || Hq <= 0 || Hkv <= 0 || D_max <= 0 || L_max <= 0) return SSD_ERR_SHAPE;
  if (Hq % Hkv != 0) return SSD_ERR_SHAPE;
  if (d != 64 && d != 128) return SSD_ERR_UNSUPPORTED;
  if (D_max > 128 || (int64_t)D_max * (Hq / Hkv) > 512) return SSD_ERR_UNSUPPORTED;
  if ((int64_t)B * Hkv > 65535) return SSD_ERR_UNSUPPORTED;
  if ((int64_t)B * Hkv * L_max >= (int64_t)1 << 31) return SSD_ERR_UNSUPPORTED;
  return SSD_OK;
}

ssd_status check_accept_common(int32_t rows, int32_t V, float temperature, const ssd_rng* rng,
                               const int32_t* out_tok, const uint8_t* accepted,
                               const int32_t* status) {
  if (rows < 0 || V <= 0) return SSD_ERR_SHAPE;
  if (rng == nullptr || out_tok == nullptr || accepted == nullptr || status == nullptr)
    return SSD_ERR_INVALID_ARG;
  if (!(temperature > 0.f) || !isfinite(temperature)) return SSD_ERR_INVALID_ARG;
  if (rng->uniforms != nullptr && (reinterpret_cast<uintptr_t>(rng->uniforms) & 7u) != 0)
    return SSD_ERR_INVALID_ARG;  // read as float2
  return SSD_OK;
}

bool strategy_ok(int32_t strategy) {
  return strategy == SSD_STRATEGY_ACCEPT_REJECT || strategy == SSD_STRATEGY_GREEDY ||
         strategy == SSD_STRATEGY_SAMPLE;
}

ssd_status check_logits(int32_t rows, int32_t V, const float* tgt, const float* drf, int64_t ld) {
  if (rows == 0) return SSD_OK;
  if (tgt == nullptr || drf == nullptr) return SSD_ERR_INVALID_ARG;
  if (V % 4 != 0 || ld % 4 != 0 || ld < V) return SSD_ERR_SHAPE;
  if (!aligned16(tgt) || !aligned16(drf)) return SSD_ERR_INVALID_ARG;
  if (!accept_supported(V)) return SSD_ERR_UNSUPPORTED;
  if ((int64_t)rows * 8 > INT32_MAX) return SSD_ERR_UNSUPPORTED;
  return SSD_OK;
}

}  // namespace

extern "C" {

int32_t ssd_abi_version(void) { return SSD_ABI_VERSION; }

void ssd_set_wait_limit(uint32_t max_polls) {
  g_wait_polls.store(max_polls, std::memory_order_relaxed);
}

void ssd_set_barrier_shortfall(uint32_t arrivals) {
  g_barrier_shortfall.store(arrivals, std::memory_order_relaxed);
}

const char* ssd_status_string(ssd_status s) {
  switch (s) {
    case SSD_OK: return "SSD_OK";
    case SSD_ERR_INVALID_ARG: return "SSD_ERR_INVALID_ARG";
    case SSD_ERR_SHAPE: return "SSD_ERR_SHAPE";
    case SSD_ERR_UNSUPPORTED: return "SSD_ERR_UNSUPPORTED";
    case SSD_ERR_CUDA: return "SSD_ERR_CUDA";
    case SSD_ERR_TIMEOUT: return "SSD_ERR_TIMEOUT";
    case SSD_ERR_DEVICE_BOUNDS: return "SSD_ERR_DEVICE_BOUNDS";
    case SSD_ERR_WORKSPACE: return "SSD_ERR_WORKSPACE";
  }
  return "SSD_ERR_UNKNOWN";
}

ssd_status ssd_frontier(const ssd_grid* grid, int32_t B, const int32_t* cache_len, int32_t D_max,
                        int32_t* n_drafts, int32_t* draft_pos, int32_t* status,
                        ssd_stream_t stream) {
  ssd_status s = check_grid(grid);
  if (s != SSD_OK) return s;
  if (grid->row_stride != grid->grid_w) return SSD_ERR_UNSUPPORTED;
  if (B < 0 || D_max <= 0) return SSD_ERR_SHAPE;
  if ((int64_t)(grid->k_v + 1) * grid->grid_w > D_max) return SSD_ERR_SHAPE;
  if (B == 0) return SSD_OK;
  if (cache_len == nullptr || n_drafts == nullptr || draft_pos == nullptr || status == nullptr)
    return SSD_ERR_INVALID_ARG;
  return from_cuda(launch_frontier(*grid, B, cache_len, D_max, n_drafts, draft_pos, status,
                                   (cudaStream_t)stream));
}

size_t ssd_verify_attention_workspace(int32_t B, int32_t Hq, int32_t Hkv, int32_t d,
                                      int32_t D_max, int32_t L_max) {
  if (B <= 0 || Hq <= 0 || Hkv <= 0 || Hq % Hkv != 0 || D_max <= 0 || L_max <= 0) return 0;
  return attention_workspace(B, Hq, Hkv, d, D_max, L_max);
}

ssd_status ssd_verify_attention(const ssd_grid* grid, int32_t B, int32_t Hq, int32_t Hkv,
                                int32_t d, const int32_t* cache_len, const int32_t* n_drafts,
                                const int32_t* draft_pos, int32_t D_max, int32_t L_max,
                                const void* q, const void* k, const void* v, float scale,
                                void* o, float* lse, void* workspace, size_t workspace_bytes,
                                int32_t* status, ssd_stream_t stream) {
  ssd_status s = check_attention(grid, B, Hq, Hkv, d, D_max, L_max);
  if (s != SSD_OK) return s;
  if (B == 0) return SSD_OK;
  if (cache_len == nullptr || n_drafts == nullptr || draft_pos == nullptr || q == nullptr ||
      k == nullptr || v == nullptr || o == nullptr || status == nullptr)
    return SSD_ERR_INVALID_ARG;
  if (!aligned16(k) || !aligned16(v) || !aligned16(q) || !aligned16(o)) return SSD_ERR_INVALID_ARG;
  if (!(scale >= 0.f) || !isfinite(scale)) return SSD_ERR_INVALID_ARG;
  const size_t need = attention_workspace(B, Hq, Hkv, d, D_max, L_max);
  if (workspace == nullptr || workspace_bytes < need) return SSD_ERR_WORKSPACE;
  AttnArgs a;
  a.grid = *grid;
  a.B = B;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.d = d;
  a.D_max = D_max;
  a.L_max = L_max;
  a.cache_len = cache_len;
  a.n_drafts = n_drafts;
  a.draft_pos = draft_pos;
  a.q = q;
  a.k = k;
  a.v = v;
  a.scale = scale;
  a.o = o;
  a.lse = lse;
  a.status = status;
  return from_cuda(launch_attention(a, workspace, workspace_bytes, (cudaStream_t)stream));
}

ssd_status ssd_verify_attention_noalloc(const ssd_grid* grid, int32_t B, int32_t Hq, int32_t Hkv,
                                        int32_t d, const int32_t* cache_len,
                                        const int32_t* n_drafts, const int32_t* draft_pos,
                                        int32_t D_max, int32_t L_max, const void* q, const void* k,
                                        const void* v, float scale, void* o, float* lse,
                                        int32_t* status, ssd_stream_t stream) {
  ssd_status s = check_attention(grid, B, Hq, Hkv, d, D_max, L_max);
  if (s != SSD_OK) return s;
  if (B == 0) return SSD_OK;
  if (cache_len == nullptr || n_drafts == nullptr || draft_pos == nullptr || q == nullptr ||
      k == nullptr || v == nullptr || o == nullptr || status == nullptr)
    return SSD_ERR_INVALID_ARG;
  if (!aligned16(k) || !aligned16(v) || !aligned16(q) || !aligned16(o)) return SSD_ERR_INVALID_ARG;
  if (!(scale >= 0.f) || !isfinite(scale)) return SSD_ERR_INVALID_ARG;
  if (attention_workspace(B, Hq, Hkv, d, D_max, L_max) > SSD_NOALLOC_SCRATCH_BYTES)
    return SSD_ERR_WORKSPACE;
  AttnArgs a;
  a.grid = *grid;
  a.B = B;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.d = d;
  a.D_max = D_max;
  a.L_max = L_max;
  a.cache_len = cache_len;
  a.n_drafts = n_drafts;
  a.draft_pos = draft_pos;
  a.q = q;
  a.k = k;
  a.v = v;
  a.scale = scale;
  a.o = o;
  a.lse = lse;
  a.status = status;
  const cudaError_t e = launch_attention_noalloc(a, (cudaStream_t)stream);
  if (e == cudaErrorMemoryAllocation) return SSD_ERR_WORKSPACE;
  return from_cuda(e);
}

ssd_status ssd_accept_strategy(int32_t strategy, int32_t rows, int32_t V, const float* tgt_logits,
                               const float* drf_logits, int64_t ld, const int32_t* draft_tok,
                               float temperature, const ssd_rng* rng, int32_t* out_tok,
                               uint8_t* accepted, float* ratio, float* lse, int32_t* status,
                               ssd_stream_t stream) {
  if (!strategy_ok(strategy)) return SSD_ERR_INVALID_ARG;
  ssd_status s = check_accept_common(rows, V, temperature, rng, out_tok, accepted, status);
  if (s != SSD_OK) return s;
  s = check_logits(rows, V, tgt_logits, drf_logits, ld);
  if (s != SSD_OK) return s;
  if (rows == 0) return SSD_OK;
  AcceptArgs a;
  a.rows = rows;
  a.V = V;
  a.tgt = tgt_logits;
  a.drf = drf_logits;
  a.ld = ld;
  a.draft_tok = draft_tok;
  a.temperature = temperature;
  a.rng = *rng;
  a.out_tok = out_tok;
  a.accepted = accepted;
  a.ratio = ratio;
  a.lse = lse;
  a.status = status;
  a.n_drafts = nullptr;
  a.D_max = 1;
  a.strategy = strategy;
  a.ref_rows = nullptr;
  a.ref_init = 0;
  a.bonus = 0;
  return from_cuda(launch_accept(a, (cudaStream_t)stream));
}

ssd_status ssd_accept_round(int32_t strategy, int32_t rows, int32_t V, const float* tgt_logits,
                            int64_t ld, const float** ref_rows, const int32_t* tok,
                            float temperature, const ssd_rng* rng, int32_t* out_tok,
                            uint8_t* accepted, float* ratio, float* lse, int32_t* status,
                            ssd_stream_t stream) {
  if (!strategy_ok(strategy)) return SSD_ERR_INVALID_ARG;
  ssd_status s = check_accept_common(rows, V, temperature, rng, out_tok, accepted, status);
  if (s != SSD_OK) return s;
  if (rows == 0) return SSD_OK;
  if (ref_rows == nullptr) return SSD_ERR_INVALID_ARG;
  // the reference rows are only known on the device; the target is checked
  // like the draft logits of ssd_accept_strategy()
  s = check_logits(rows, V, tgt_logits, tgt_logits, ld);
  if (s != SSD_OK) return s;
  AcceptArgs a;
  a.rows = rows;
  a.V = V;
  a.tgt = tgt_logits;
  a.drf = nullptr;
  a.ld = ld;
  a.draft_tok = tok;
  a.temperature = temperature;
  a.rng = *rng;
  a.out_tok = out_tok;
  a.accepted = accepted;
  a.ratio = ratio;
  a.lse = lse;
  a.status = status;
  a.n_drafts = nullptr;
  a.D_max = 1;
  a.strategy = strategy;
  a.ref_rows = ref_rows;
  a.ref_init = 0;
  a.bonus = 0;
  return from_cuda(launch_accept(a, (cudaStream_t)stream));
}

size_t ssd_draft_predict_workspace(int32_t rows, int32_t d, int32_t m, int32_t V) {
  if (rows <= 0 || d <= 0 || m <= 0 || V <= 0) return 0;
  return predictor_workspace(rows, d, m, V, true);
}

ssd_status ssd_draft_predict(int32_t rows, int32_t d, int32_t m, int32_t V, const void* z,
                             const void* w0, const void* w1, const void* w3, const void* w2,
                             const float* gamma1, const float* gamma2, const void* w_head,
                             float eps, int32_t* out_tok, float* out_hidden, void* workspace,
                             size_t workspace_bytes, int32_t* status, ssd_stream_t stream) {
  if (rows <= 0 || d <= 0 || m <= 0 || V <= 0) return SSD_ERR_SHAPE;
  if (d % 8 != 0 || m % 8 != 0 || V % 4 != 0) return SSD_ERR_SHAPE;
  if (!predictor_supported(d, m, V)) return SSD_ERR_UNSUPPORTED;
  if ((int64_t)rows * 2 * d >= (int64_t)1 << 31 || (int64_t)rows * m >= (int64_t)1 << 31)
    return SSD_ERR_UNSUPPORTED;
  const void* ptrs[] = {z, w0, w1, w3, w2, gamma1, gamma2, w_head, out_tok, status};
  for (const void* q : ptrs)
    if (q == nullptr) return SSD_ERR_INVALID_ARG;
  for (const void* q : {z, w0, w1, w3, w2, w_head, (const void*)gamma1, (const void*)gamma2,
                        (const void*)out_hidden})
    if (q != nullptr && !aligned16(q)) return SSD_ERR_INVALID_ARG;
  if (!(eps >= 0.f) || !isfinite(eps)) return SSD_ERR_INVALID_ARG;
  if (workspace == nullptr ||
      workspace_bytes < predictor_workspace(rows, d, m, V, out_hidden == nullptr))
    return SSD_ERR_WORKSPACE;
  PredictorArgs p;
  p.rows = rows;
  p.d = d;
  p.m = m;
  p.V = V;
  p.z = z;
  p.w0 = w0;
  p.w1 = w1;
  p.w3 = w3;
  p.w2 = w2;
  p.gamma1 = gamma1;
  p.gamma2 = gamma2;
  p.w_head = w_head;
  p.eps = eps;
  p.out_tok = out_tok;
  p.out_hidden = out_hidden;
  return from_cuda(launch_predictor(p, workspace, workspace_bytes, status, (cudaStream_t)stream));
}

ssd_status ssd_commit_pass(const ssd_grid* grid, int32_t B, const int32_t* cache_len,
                           int32_t D_max, int32_t commit, int32_t* next_cache_len,
                           int32_t* status, ssd_stream_t stream) {
  ssd_status s = check_grid(grid);
  if (s != SSD_OK) return s;
  if (grid->row_stride != grid->grid_w) return SSD_ERR_UNSUPPORTED;
  if (commit != SSD_COMMIT_NONE && commit != SSD_COMMIT_BLOCK && commit != SSD_COMMIT_FIRST_ROW)
    return SSD_ERR_INVALID_ARG;
  if (B < 0 || D_max <= 0) return SSD_ERR_SHAPE;
  if ((int64_t)(grid->k_v + 1) * grid->grid_w > D_max) return SSD_ERR_SHAPE;
  if (B == 0) return SSD_OK;
  if (cache_len == nullptr || next_cache_len == nullptr || status == nullptr)
    return SSD_ERR_INVALID_ARG;
  return from_cuda(launch_commit(*grid, commit, B, D_max, cache_len, next_cache_len, status,
                                 (cudaStream_t)stream));
}

ssd_status ssd_record_commit(int32_t B, int32_t D_max, int32_t prefix_len, int32_t hw,
                             const int32_t* cache_len, const int32_t* next_cache_len,
                             const int32_t* out_tok, int32_t* grid_tok, int32_t* status,
                             ssd_stream_t stream) {
  if (B < 0 || D_max <= 0 || prefix_len < 0 || hw <= 0) return SSD_ERR_SHAPE;
  if (B == 0) return SSD_OK;
  if (cache_len == nullptr || next_cache_len == nullptr || out_tok == nullptr ||
      grid_tok == nullptr || status == nullptr)
    return SSD_ERR_INVALID_ARG;
  return from_cuda(launch_record_commit(B, D_max, prefix_len, hw, cache_len, next_cache_len,
                                        out_tok, grid_tok, status, (cudaStream_t)stream));
}

ssd_status ssd_stage_shift(int32_t B, int32_t D_max, int32_t W, int32_t* tok,
                           const float** ref_rows, ssd_stream_t stream) {
  if (B < 0 || D_max <= 0 || W < 0 || 2 * (int64_t)W > D_max) return SSD_ERR_SHAPE;
  if (B == 0 || W == 0) return SSD_OK;
  if (tok == nullptr) return SSD_ERR_INVALID_ARG;
  return from_cuda(launch_stage_shift(B, D_max, W, tok, ref_rows, (cudaStream_t)stream));
}

ssd_status ssd_accept(int32_t rows, int32_t V, const float* tgt_logits, const float* drf_logits,
                      int64_t ld, const int32_t* draft_tok, float temperature, const ssd_rng* rng,
                      int32_t* out_tok, uint8_t* accepted, float* ratio, float* lse,
                      int32_t* status, ssd_stream_t stream) {
  return ssd_accept_strategy(SSD_STRATEGY_ACCEPT_REJECT, rows, V, tgt_logits, drf_logits, ld,
                             draft_tok, temperature, rng, out_tok, accepted, ratio, lse, status,
                             stream);
}

size_t ssd_lmhead_accept_workspace(int32_t rows, int32_t V) {
  if (rows <= 0 || V <= 0) return 0;
  return lmhead_workspace(rows, V);
}

ssd_status ssd_lmhead_accept(int32_t rows, int32_t V, int32_t K, const void* h_tgt,
                             const void* h_drf, const void* w_tgt, const void* w_drf,
                             const int32_t* draft_tok, float temperature, const ssd_rng* rng,
                             int32_t* out_tok, uint8_t* accepted, float* ratio, float* lse,
                             void* workspace, size_t workspace_bytes, int32_t* status,
                             ssd_stream_t stream) {
  ssd_status s = check_accept_common(rows, V, temperature, rng, out_tok, accepted, status);
  if (s != SSD_OK) return s;
  if (rows == 0) return SSD_OK;
  s = lmhead_check(rows, V, K);
  if (s != SSD_OK) return s;
  if (h_tgt == nullptr || h_drf == nullptr || w_tgt == nullptr || w_drf == nullptr)
    return SSD_ERR_INVALID_ARG;
  if (!aligned16(h_tgt) || !aligned16(h_drf) || !aligned16(w_tgt) || !aligned16(w_drf))
    return SSD_ERR_INVALID_ARG;
  if (workspace == nullptr || workspace_bytes < lmhead_workspace(rows, V)) return SSD_ERR_WORKSPACE;
  LmHeadArgs a;
  a.rows = rows;
  a.V = V;
  a.K = K;
  a.h_tgt = h_tgt;
  a.h_drf = h_drf;
  a.w_tgt = w_tgt;
  a.w_drf = w_drf;
  a.draft_tok = draft_tok;
  a.temperature = temperature;
  a.rng = *rng;
  a.out_tok = out_tok;
  a.accepted = accepted;
  a.ratio = ratio;
  a.lse = lse;
  a.status = status;
  a.n_drafts = nullptr;
  a.D_max = 1;
  return from_cuda(launch_lmhead(a, workspace, workspace_bytes, (cudaStream_t)stream));
}

}  // extern "C"

namespace {

// Strategy (C) under a prefix rule, one round, from logits: only the tokens
// the counts commit are drawn (AcceptArgs::lazy).
bool lazy_draws(const ssd_verify_args* x) {
  return x->tgt_logits != nullptr && x->strategy == SSD_STRATEGY_ACCEPT_REJECT &&
         x->ref_rows == nullptr &&
         (x->commit == SSD_COMMIT_PREFIX || x->commit == SSD_COMMIT_PREFIX_BONUS);
}

// Workspace of the acceptance part (a3-a7) of a step.  Fused path: the
// lm_head's.  Logits path: the per-row normalisers of a lazy pass, a ticket
// per sequence and the block masses of the committed rows, counted under
// every strategy and commit rule so that one workspace serves any mode.
struct AcceptWs {
  float2* stats;
  int32_t* tickets;
  float* mass;
};
size_t accept_part_workspace(const ssd_verify_args* x) {
  if (x->tgt_logits == nullptr && x->w_tgt != nullptr)
    return align256(ssd_lmhead_accept_workspace(x->B * x->D_max, x->V));
  return align256((size_t)x->B * x->D_max * sizeof(float2)) +
         align256((size_t)x->B * sizeof(int32_t)) +
         align256((size_t)x->B * resolve_blocks(x->V) * sizeof(float));
}
AcceptWs carve_accept(const ssd_verify_args* x, void* ws) {
  unsigned char* w = static_cast<unsigned char*>(ws);
  AcceptWs c;
  c.stats = reinterpret_cast<float2*>(w);
  w += align256((size_t)x->B * x->D_max * sizeof(float2));
  c.tickets = reinterpret_cast<int32_t*>(w);
  w += align256((size_t)x->B * sizeof(int32_t));
  c.mass = reinterpret_cast<float*>(w);
  return c;
}

// Argument checks of the acceptance part, shared by ssd_verify_step and
// ssd_verify_accept (shapes of the grid and the batch checked by the caller).
ssd_status check_accept_part(const ssd_verify_args* x, const ssd_verify_out* y) {
  if (x->cache_len == nullptr) return SSD_ERR_INVALID_ARG;
  if (y->n_drafts == nullptr || y->draft_pos == nullptr || y->out_tok == nullptr ||
      y->accepted == nullptr || y->accepted_count == nullptr || y->accepted_prefix == nullptr ||
      y->next_cache_len == nullptr || y->status == nullptr)
    return SSD_ERR_INVALID_ARG;
  const int32_t rows = x->B * x->D_max;
  ssd_status s =
      check_accept_common(rows, x->V, x->temperature, &x->rng, y->out_tok, y->accepted, y->status);
  if (s != SSD_OK) return s;
  if (!strategy_ok(x->strategy)) return SSD_ERR_INVALID_ARG;
  if (x->commit < SSD_COMMIT_PREFIX || x->commit > SSD_COMMIT_PREFIX_BONUS) return SSD_ERR_INVALID_ARG;
  if (x->ref_init != 0 && (x->ref_rows == nullptr || x->drf_logits == nullptr))
    return SSD_ERR_INVALID_ARG;
  if (x->tgt_logits == nullptr) {
    if (x->h_tgt == nullptr || x->h_drf == nullptr || x->w_tgt == nullptr || x->w_drf == nullptr)
      return SSD_ERR_INVALID_ARG;
    if (x->strategy != SSD_STRATEGY_ACCEPT_REJECT || x->ref_rows != nullptr ||
        x->commit == SSD_COMMIT_PREFIX_BONUS)
      return SSD_ERR_UNSUPPORTED;
    return lmhead_check(rows, x->V, x->hidden);
  }
  return check_logits(rows, x->V, x->tgt_logits, x->drf_logits, x->ld);
}

// Logits path, a1 + a3-a5: the acceptance pass, which computes the frontier
// itself and writes it out (n_drafts, draft_pos).
#ifndef SSD_ACCEPT_EARLY_PDL
#define SSD_ACCEPT_EARLY_PDL 1
#endif

cudaError_t launch_accept_phase(const ssd_verify_args* x, const ssd_verify_out* y, void* ws,
                                cudaStream_t stream, int early_dependents = 0) {
  const bool lazy = lazy_draws(x);
  const AcceptWs w = carve_accept(x, ws);
  AcceptArgs c;
  c.rows = x->B * x->D_max;
  c.V = x->V;
  c.tgt = x->tgt_logits;
  c.drf = x->drf_logits;
  c.ld = x->ld;
  c.draft_tok = x->draft_tok;
  c.temperature = x->temperature;
  c.rng = x->rng;
  c.out_tok = y->out_tok;
  c.accepted = y->accepted;
  c.ratio = y->ratio;
  c.lse = nullptr;
  c.status = y->status;
  c.n_drafts = nullptr;
  c.D_max = x->D_max;
  c.strategy = x->strategy;
  c.ref_rows = x->ref_rows;
  c.ref_init = x->ref_init;
  c.bonus = x->commit == SSD_COMMIT_PREFIX_BONUS;
  c.lazy = lazy ? 1 : 0;
  c.stats = lazy ? w.stats : nullptr;
  c.cache_len = x->cache_len;
  c.grid = x->grid;
  c.n_drafts_out = y->n_drafts;
  c.draft_pos = y->draft_pos;
  c.tickets = w.tickets;
  c.early_dependents = early_dependents;
  return launch_accept(c, stream);
}

// Logits path, a7: the counts, with the committed draws after a lazy pass.
cudaError_t launch_finish_phase(const ssd_verify_args* x, const ssd_verify_out* y, void* ws,
                                bool pdl, cudaStream_t stream) {
  if (!lazy_draws(x))
    return launch_counts(x->grid, x->commit, x->B, x->D_max, x->cache_len, y->n_drafts,
                         y->accepted, y->accepted_count, y->accepted_prefix, y->next_cache_len,
                         y->status, pdl, stream);
  const AcceptWs w = carve_accept(x, ws);
  ResolveArgs r;
  r.grid = x->grid;
  r.commit = x->commit;
  r.B = x->B;
  r.D_max = x->D_max;
  r.V = x->V;
  r.tgt = x->tgt_logits;
  r.drf = x->drf_logits;
  r.ld = x->ld;
  r.temperature = x->temperature;
  r.rng = x->rng;
  r.cache_len = x->cache_len;
  r.n_drafts = y->n_drafts;
  r.stats = w.stats;
  r.bonus = x->commit == SSD_COMMIT_PREFIX_BONUS;
  r.out_tok = y->out_tok;
  r.accepted = y->accepted;
  r.accepted_count = y->accepted_count;
  r.accepted_prefix = y->accepted_prefix;
  r.next_cache_len = y->next_cache_len;
  r.status = y->status;
  r.tickets = w.tickets;
  r.mass = w.mass;
  return launch_resolve(r, pdl, stream);
}

// Fused path, a1 + a6 + a7 on one stream (the frontier already written).
cudaError_t launch_fused_accept(const ssd_verify_args* x, const ssd_verify_out* y, void* ws,
                                size_t ws_bytes, cudaStream_t stream) {
  LmHeadArgs h;
  h.rows = x->B * x->D_max;
  h.V = x->V;
  h.K = x->hidden;
  h.h_tgt = x->h_tgt;
  h.h_drf = x->h_drf;
  h.w_tgt = x->w_tgt;
  h.w_drf = x->w_drf;
  h.draft_tok = x->draft_tok;
  h.temperature = x->temperature;
  h.rng = x->rng;
  h.out_tok = y->out_tok;
  h.accepted = y->accepted;
  h.ratio = y->ratio;
  h.lse = nullptr;
  h.status = y->status;
  h.n_drafts = y->n_drafts;
  h.D_max = x->D_max;
  // a one-round prefix commit keeps one drawn token per sequence: draw only it
  h.lazy = x->commit == SSD_COMMIT_PREFIX ? 1 : 0;
  h.counters_zeroed = 1;  // by the frontier kernel before it
  cudaError_t e = launch_lmhead(h, ws, ws_bytes, stream);
  if (e != cudaSuccess) return e;
  return launch_counts(x->grid, x->commit, x->B, x->D_max, x->cache_len, y->n_drafts, y->accepted,
                       y->accepted_count, y->accepted_prefix, y->next_cache_len, y->status,
                       false, stream);
}

}  // namespace

extern "C" {

size_t ssd_verify_step_workspace(const ssd_verify_args* x) {
  if (x == nullptr || x->B <= 0) return 0;
  return align256(ssd_verify_attention_workspace(x->B, x->Hq, x->Hkv, x->d, x->D_max, x->L_max)) +
         accept_part_workspace(x);
}

int32_t ssd_verify_step_launches(const ssd_verify_args* x) {
  if (x == nullptr) return -1;
  if (check_attention(&x->grid, x->B, x->Hq, x->Hkv, x->d, x->D_max, x->L_max) != SSD_OK) return -1;
  if (x->B == 0) return 0;
  // logits: acceptance (with the frontier) + attention (+ split combine) + counts/draws;
  // fused: frontier + attention (+ combine) + lm_head acceptance + counts
  const int fixed = x->tgt_logits != nullptr ? 2 : 3;
  return fixed + attention_launches(x->grid, x->B, x->Hq, x->Hkv, x->d, x->D_max, x->L_max);
}

ssd_status ssd_verify_step(const ssd_verify_args* x, const ssd_verify_out* y, void* workspace,
                           size_t workspace_bytes, ssd_stream_t stream_) {
  if (x == nullptr || y == nullptr) return SSD_ERR_INVALID_ARG;
  cudaStream_t stream = (cudaStream_t)stream_;
  ssd_status s = check_attention(&x->grid, x->B, x->Hq, x->Hkv, x->d, x->D_max, x->L_max);
  if (s != SSD_OK) return s;
  if (x->grid.row_stride != x->grid.grid_w) return SSD_ERR_UNSUPPORTED;
  if ((int64_t)(x->grid.k_v + 1) * x->grid.grid_w > x->D_max) return SSD_ERR_SHAPE;
  if (x->B == 0) return SSD_OK;
  if (x->q == nullptr || x->k == nullptr || x->v == nullptr) return SSD_ERR_INVALID_ARG;
  if (y->draft_pos == nullptr || y->o == nullptr) return SSD_ERR_INVALID_ARG;
  s = check_accept_part(x, y);
  if (s != SSD_OK) return s;
  // The counts write next_cache_len while the attention (beside them, or as
  // the kernel they depend on programmatically) may still read cache_len.
  {
    const uintptr_t c0 = (uintptr_t)x->cache_len, n0 = (uintptr_t)y->next_cache_len;
    const uintptr_t len = (uintptr_t)x->B * sizeof(int32_t);
    if (c0 < n0 + len && n0 < c0 + len) return SSD_ERR_INVALID_ARG;
  }
  if (!(x->scale >= 0.f) || !isfinite(x->scale)) return SSD_ERR_INVALID_ARG;
  const size_t need = ssd_verify_step_workspace(x);
  if (workspace == nullptr || workspace_bytes < need) return SSD_ERR_WORKSPACE;
  unsigned char* ws = static_cast<unsigned char*>(workspace);
  const size_t attn_ws = align256(attention_workspace(x->B, x->Hq, x->Hkv, x->d, x->D_max, x->L_max));
  AttnArgs a;
  a.grid = x->grid;
  a.B = x->B;
  a.Hq = x->Hq;
  a.Hkv = x->Hkv;
  a.d = x->d;
  a.D_max = x->D_max;
  a.L_max = x->L_max;
  a.cache_len = x->cache_len;
  a.n_drafts = y->n_drafts;
  a.draft_pos = y->draft_pos;
  a.q = x->q;
  a.k = x->k;
  a.v = x->v;
  a.scale = x->scale;
  a.o = y->o;
  a.lse = y->lse;
  a.status = y->status;
  cudaError_t e;
  SideStream* side = nullptr;
  if (x->tgt_logits != nullptr) {
    // Logits path: the acceptance pass computes the frontier and writes it
    // out (a1 + a3-a5); the attention computes the same frontier from
    // cache_len (a2), so the two need no frontier launch before them.
    a.raster = 1;
    // Rows that can hold a draft: the frontier bound per sequence (+ the bonus row).
    const int64_t live_rows =
        (int64_t)x->B * std::min<int32_t>(x->D_max, attention_rows_hint(x->grid, x->D_max) +
                                                        (x->commit == SSD_COMMIT_PREFIX_BONUS));
    // Measured on GB300: lazy (C) gains from hiding its draws under the attention; greedy,
    // which has nothing to hide, gains from this order only when its pass is short (few
    // live rows, e.g. the horizontal stage: 33.4 -> 31.5 us), and loses on the sweep.
    const bool serial =
        x->B * x->D_max >= 2 * device_sm_count() &&
        (lazy_draws(x) || (x->strategy == SSD_STRATEGY_GREEDY && live_rows <= device_sm_count()));
    if (serial) {
      // On `stream` alone: the acceptance; the attention, which reads none of
      // its results, as a programmatic dependent (the tcgen05 kernel starts
      // as the acceptance's CTAs retire and lets the next kernel be scheduled
      // only once the acceptance has completed; the mma.sync kernel starts
      // after it); then a7 (the counts, with the committed draws when lazy) as
      // a programmatic dependent of the attention: its small CTAs run beside
      // the attention, in the registers it leaves free.
      e = launch_accept_phase(x, y, ws + attn_ws, stream, /*early_dependents=*/SSD_ACCEPT_EARLY_PDL);
      if (e != cudaSuccess) return SSD_ERR_CUDA;
      e = launch_attention(a, ws, attn_ws, stream, /*defer_combine=*/true, /*pdl=*/true);
      if (e != cudaSuccess) return SSD_ERR_CUDA;
      e = launch_finish_phase(x, y, ws + attn_ws, /*pdl=*/true, stream);
      if (e != cudaSuccess) return SSD_ERR_CUDA;
      return from_cuda(launch_attention_combine(a, ws, stream));
    }
    // Otherwise the acceptance and a7 on a side stream beside the attention:
    // kernels that do not fill the GPU, or that draw every row, overlap.
    if (side_stream(&side) != cudaSuccess) return SSD_ERR_CUDA;
    if (cudaEventRecord(side->fork, stream) != cudaSuccess ||
        cudaStreamWaitEvent(side->stream, side->fork, 0) != cudaSuccess)
      return SSD_ERR_CUDA;
    // (the attention first: its persistent CTAs deal their items statically,
    // while the acceptance's rows adapt to CTAs that start late)
    e = launch_attention(a, ws, attn_ws, stream);
    if (e != cudaSuccess) return SSD_ERR_CUDA;
    e = launch_accept_phase(x, y, ws + attn_ws, side->stream);
    if (e != cudaSuccess) return SSD_ERR_CUDA;
    e = launch_finish_phase(x, y, ws + attn_ws, /*pdl=*/false, side->stream);
    if (e != cudaSuccess) return SSD_ERR_CUDA;
    if (cudaEventRecord(side->join, side->stream) != cudaSuccess ||
        cudaStreamWaitEvent(stream, side->join, 0) != cudaSuccess)
      return SSD_ERR_CUDA;
    return SSD_OK;
  }
  // Fused path: a1, then the attention on `stream` beside the lm_head
  // acceptance and the counts on a side stream, joined back into `stream`.
  if (side_stream(&side) != cudaSuccess) return SSD_ERR_CUDA;
  e = launch_frontier(x->grid, x->B, x->cache_len, x->D_max, y->n_drafts, y->draft_pos, y->status,
                      stream, lmhead_counters(ws + attn_ws), kLmheadCounters);
  if (e != cudaSuccess) return SSD_ERR_CUDA;
  if (cudaEventRecord(side->fork, stream) != cudaSuccess ||
      cudaStreamWaitEvent(side->stream, side->fork, 0) != cudaSuccess)
    return SSD_ERR_CUDA;
  e = launch_attention(a, ws, attn_ws, stream);
  if (e != cudaSuccess) return SSD_ERR_CUDA;
  e = launch_fused_accept(x, y, ws + attn_ws, workspace_bytes - attn_ws, side->stream);
  if (e != cudaSuccess) return SSD_ERR_CUDA;
  if (cudaEventRecord(side->join, side->stream) != cudaSuccess ||
      cudaStreamWaitEvent(stream, side->join, 0) != cudaSuccess)
    return SSD_ERR_CUDA;
  return SSD_OK;
}

ssd_status ssd_verify_accept(const ssd_verify_args* x, const ssd_verify_out* y, void* workspace,
                             size_t workspace_bytes, ssd_stream_t stream) {
  if (x == nullptr || y == nullptr) return SSD_ERR_INVALID_ARG;
  ssd_status s = check_grid(&x->grid);
  if (s != SSD_OK) return s;
  if (x->B < 0 || x->D_max <= 0) return SSD_ERR_SHAPE;
  if (x->grid.row_stride != x->grid.grid_w) return SSD_ERR_UNSUPPORTED;
  if ((int64_t)(x->grid.k_v + 1) * x->grid.grid_w > x->D_max) return SSD_ERR_SHAPE;
  if (x->B == 0) return SSD_OK;
  s = check_accept_part(x, y);
  if (s != SSD_OK) return s;
  const size_t need = accept_part_workspace(x);
  if (workspace == nullptr || workspace_bytes < need) return SSD_ERR_WORKSPACE;
  cudaStream_t st = (cudaStream_t)stream;
  if (x->tgt_logits == nullptr) {
    cudaError_t e = launch_frontier(x->grid, x->B, x->cache_len, x->D_max, y->n_drafts,
                                    y->draft_pos, y->status, st, lmhead_counters(workspace),
                                    kLmheadCounters);
    if (e != cudaSuccess) return SSD_ERR_CUDA;
    return from_cuda(launch_fused_accept(x, y, workspace, workspace_bytes, st));
  }
  cudaError_t e = launch_accept_phase(x, y, workspace, st);
  if (e != cudaSuccess) return SSD_ERR_CUDA;
  return from_cuda(launch_finish_phase(x, y, workspace, /*pdl=*/false, st));
}

}  // extern "C"
