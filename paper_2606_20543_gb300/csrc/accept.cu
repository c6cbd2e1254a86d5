// accept.cu — vocabulary-wide acceptance (steps a3-a5): target/draft softmax,
// the ratio at the draft token, the accept decision and, on rejection, the
// residual draw (Sec. 3.3 "Verification as Auto Correction", strategy (C)):
//   accept t with probability min(p(t) / q(t), 1); otherwise draw from
//   [p - q]_+ / sum [p - q]_+ (inverse CDF in vocabulary order, one uniform).
// The same kernel runs the paper's other two strategies: (A) greedy, the
// argmax of p (tracked in the first pass), and (B) sampling, a draw from p
// (the second pass with the weights of p); under both a row is "accepted"
// when the selected token is the draft token.
//
// Design (GB300): a persistent grid of four CTAs per SM, each walking rows
// blockIdx.x, blockIdx.x + gridDim.x, ...  A dedicated producer warp streams
// every row with bulk TMA copies, 256 entries per consumer warp of both logit
// rows per stage, through a shared-memory ring: once from HBM for the
// statistics, and, when the kernel draws the residual tokens itself, once
// more (from L2, microseconds later) for the draw; it runs ahead into the next
// row while the consumers finish the current one.  Under (A), and in a
// one-round prefix-commit step (lazy: only the committed tokens are drawn, by
// resolve_kernel below), every row is streamed once.  The consumers are latency-bound, so the arithmetic is kept
// short: per first-pass chunk each thread folds its 8 entries of both rows
// into online (max, sum of 2^x) statistics with a branch-free rescale,
// three-input maxima and packed fp32 pairs (fma/add .f32x2) for the exponent
// arguments and the sums, and tracks the first argmax of q with the target
// logit at it.  A fixed-order reduction (xor tree in each warp, then a
// three-level tree over the warps) gives the log-sum-exps and the draft
// token, and one thread takes the decision with the row's uniforms drawn
// before the row's data arrived.  For rejected rows the second-pass chunks
// give the residual weights and the mass of every 256-entry block in
// vocabulary order; warp 0 scans the block masses, finds the block holding
// u_res * Z and re-walks it to pick the token.  Accepted rows only release
// their second-pass chunks.
#include <algorithm>

#include "kernels.cuh"

namespace ssd {

namespace {

#ifndef SSD_ACCEPT_CWARPS
#define SSD_ACCEPT_CWARPS 8
#endif
#ifndef SSD_ACCEPT_STAGES
#define SSD_ACCEPT_STAGES 3
#endif
#ifndef SSD_ACCEPT_CTAS
#define SSD_ACCEPT_CTAS 4
#endif
constexpr int kCWarps = SSD_ACCEPT_CWARPS;    // consumer warps
constexpr int kConsumers = kCWarps * 32;
constexpr int kThreads = kConsumers + 32;     // + the producer warp
// Entries of each row per ring stage.  Pass A gives every consumer thread two
// float4 of each row per chunk and pass B gives every consumer warp one
// 256-entry block per chunk, so a chunk is exactly 256 entries per warp.
constexpr int kChunk = 256 * kCWarps;
constexpr int kStages = SSD_ACCEPT_STAGES;
constexpr int kCtasPerSm = SSD_ACCEPT_CTAS;
static_assert(kChunk == 2 * 4 * kConsumers, "pass A covers two float4 per thread per chunk");
static_assert(kCWarps == 4 || kCWarps == 8, "consumer warps");
constexpr int kMaxV = 1 << 20;                // block-mass table: V / 128 floats of shared memory
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// Barrier among the consumer warps only (the producer warp never joins it).
__device__ __forceinline__ void consumers_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(kConsumers) : "memory");
}

__device__ __forceinline__ bool better_arg(float v, int32_t i, float bv, int32_t bi) {
  return v > bv || (v == bv && (uint32_t)i < (uint32_t)bi);
}

// Merge two (max, sum) pairs.
__device__ __forceinline__ void merge(float& m, float& s, float m2, float s2, float c) {
  const float mn = fmaxf(m, m2);
  if (mn == -INFINITY) return;
  s = s * ex2_approx((m - mn) * c) + s2 * ex2_approx((m2 - mn) * c);
  m = mn;
}

// Residual weights of 4 entries: [p - q]_+ with p = 2^(x_p c - Cp), q = 2^(x_q c - Cq),
// or p itself for the draw from p.  cc = (c, c), ncp = (-Cp, -Cp), ncq = (-Cq, -Cq).
__device__ __forceinline__ float4 weights4(const float4& xp, const float4& xq, float2 cc,
                                           float2 ncp, float2 ncq, bool from_p) {
  const float2 a0 = ffma2(make_float2(xp.x, xp.y), cc, ncp);
  const float2 a1 = ffma2(make_float2(xp.z, xp.w), cc, ncp);
  float4 w;
  if (from_p) {
    w.x = ex2_approx(a0.x);
    w.y = ex2_approx(a0.y);
    w.z = ex2_approx(a1.x);
    w.w = ex2_approx(a1.y);
  } else {
    const float2 b0 = ffma2(make_float2(xq.x, xq.y), cc, ncq);
    const float2 b1 = ffma2(make_float2(xq.z, xq.w), cc, ncq);
    w.x = fmaxf(ex2_approx(a0.x) - ex2_approx(b0.x), 0.f);
    w.y = fmaxf(ex2_approx(a0.y) - ex2_approx(b0.y), 0.f);
    w.z = fmaxf(ex2_approx(a1.x) - ex2_approx(b1.x), 0.f);
    w.w = fmaxf(ex2_approx(a1.y) - ex2_approx(b1.y), 0.f);
  }
  return w;
}

// Sum of 2^(x c - mc) over 8 entries, as a pair of partial sums.
__device__ __forceinline__ float2 exp_sum8(const float4& x0, const float4& x1, float2 cc,
                                           float2 nmc) {
  const float2 a0 = ffma2(make_float2(x0.x, x0.y), cc, nmc);
  const float2 a1 = ffma2(make_float2(x0.z, x0.w), cc, nmc);
  const float2 a2 = ffma2(make_float2(x1.x, x1.y), cc, nmc);
  const float2 a3 = ffma2(make_float2(x1.z, x1.w), cc, nmc);
  const float2 e0 = make_float2(ex2_approx(a0.x), ex2_approx(a0.y)), e1 = make_float2(ex2_approx(a1.x), ex2_approx(a1.y));
  const float2 e2 = make_float2(ex2_approx(a2.x), ex2_approx(a2.y)), e3 = make_float2(ex2_approx(a3.x), ex2_approx(a3.y));
  return fadd2(fadd2(e0, e1), fadd2(e2, e3));
}

struct Shared {
  uint64_t full[kStages], empty[kStages];
  float red[kCWarps][5];
  int32_t red_i[kCWarps];
  float red_pm[kCWarps];  // greedy: per-warp maximum of p and its first index
  int32_t red_pi[kCWarps];
  int32_t t_hat;          // sampling: the draft token, for the accepted flag
  float Cp, Cq;      // log2-domain normalisers: max * c + log2(sum)
  int32_t accept;    // 1 accepted, 0 rejected, 2 no valid draft token, 3 drawn
  float u_res;
  float xp_t, xq_t;  // logits at a caller-given draft token (pass A)
};

// Rows that stream: frontier rows with an in-range (or absent) draft token
// (kind 0) and, in the horizontal stage, the bonus row after a sequence's
// last draft (kind 3).  Producer and consumers walk the same rows and skip
// the same ones.
__device__ __forceinline__ int row_kind(const AcceptArgs& a, int64_t r) {
  if (a.cache_len != nullptr || a.n_drafts != nullptr) {
    const int32_t b = (int32_t)(r / a.D_max), j = (int32_t)(r % a.D_max);
    const int32_t n = a.cache_len != nullptr ? frontier_drafts(a.grid, a.cache_len[b], a.D_max)
                                             : a.n_drafts[b];
    if (j >= n) return (a.bonus && j == n && n > 0) ? 3 : 1;  // bonus row / padding slot
  }
  if (a.draft_tok != nullptr) {
    const int32_t t = a.draft_tok[r];
    if (t < 0 || t >= a.V) return 2;   // draft token out of range
  }
  return 0;
}

// Block of 256 entries (64 float4) inside a ring chunk, one per consumer warp:
// warp w holds the chunk's float4 w * 64 + lane (first half of the block) and
// w * 64 + 32 + lane (second half).
constexpr int kBlocksPerChunk = kChunk / 256;  // one per consumer warp
static_assert(kBlocksPerChunk == kCWarps, "pass B: one block per consumer warp per chunk");
// Initial running maximum: finite, so exp2 arguments never meet (-inf) - (-inf).
constexpr float kLowest = -1.0e30f;

// Scan the block masses in vocabulary order (warp 0): returns the block
// holding target = u * Z and the remaining target inside it (INF: take the
// last positive entry), or -1 if Z == 0.
__device__ __forceinline__ int32_t find_block(const float* mass, int32_t nblocks, float u,
                                              float* t_in_block, int lane) {
  const int32_t per = (nblocks + 31) / 32;
  float ls = 0.f;
  for (int32_t q = 0; q < per; ++q) {
    const int32_t bk = lane * per + q;
    ls += (bk < nblocks) ? mass[bk] : 0.f;
  }
  float incl = ls;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  const float Z = __shfl_sync(0xffffffffu, incl, 31);
  if (!(Z > 0.f)) return -1;
  const float target = u * Z;
  const uint32_t pos = __ballot_sync(0xffffffffu, ls > 0.f);
  const uint32_t cross = __ballot_sync(0xffffffffu, ls > 0.f && incl > target);
  const int32_t ls_star = cross ? (__ffs(cross) - 1) : (31 - __clz(pos));
  float t1 = __shfl_sync(0xffffffffu, incl - ls, ls_star);
  t1 = cross ? target - t1 : INFINITY;
  int32_t bs = -1, blast = -1;
  float tb = INFINITY;
  if (lane == ls_star) {
    float cum = 0.f;
    for (int32_t q = 0; q < per; ++q) {
      const int32_t bk = lane * per + q;
      const float m = (bk < nblocks) ? mass[bk] : 0.f;
      if (m > 0.f) {
        blast = bk;
        if (bs < 0 && cum + m > t1) { bs = bk; tb = t1 - cum; }
      }
      cum += m;
    }
    if (bs < 0) { bs = blast; tb = INFINITY; }
  }
  bs = __shfl_sync(0xffffffffu, bs, ls_star);
  *t_in_block = __shfl_sync(0xffffffffu, tb, ls_star);
  return bs;
}

// Warp-wide scan of one 128-entry span whose lane l holds the residual
// weights w of entries e .. e + 3 (e ascending with l).  If the target th
// falls inside the span's mass, returns the token at the crossing; otherwise
// returns -1 and leaves the span's mass in *hsum.  *last_pos is updated to
// the last entry with positive weight seen so far.
__device__ __forceinline__ int32_t walk_half(const float4& w, int32_t e, float th, float* hsum,
                                             int32_t* last_pos, int lane) {
  const float lsum = (w.x + w.y) + (w.z + w.w);
  float li = lsum;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float y = __shfl_up_sync(0xffffffffu, li, o);
    if (lane >= o) li += y;
  }
  *hsum = __shfl_sync(0xffffffffu, li, 31);
  int32_t lp = -1;  // last entry of this lane with positive weight
  if (w.w > 0.f) lp = e + 3; else if (w.z > 0.f) lp = e + 2;
  else if (w.y > 0.f) lp = e + 1; else if (w.x > 0.f) lp = e;
  const uint32_t hasp = __ballot_sync(0xffffffffu, lp >= 0);
  if (hasp) *last_pos = __shfl_sync(0xffffffffu, lp, 31 - __clz(hasp));
  if (!(*hsum > 0.f && th < *hsum)) return -1;
  const uint32_t lcross = __ballot_sync(0xffffffffu, lsum > 0.f && li > th);
  const int32_t lstar = lcross ? (__ffs(lcross) - 1) : (31 - __clz(hasp));
  int32_t pick = -1;
  if (lane == lstar) {
    const float t4 = th - (li - lsum);
    const float ws[4] = {w.x, w.y, w.z, w.w};
    float acc = 0.f;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      acc += ws[k];
      if (pick < 0 && ws[k] > 0.f && acc > t4) pick = e + k;
    }
    if (pick < 0) pick = lp;
  }
  return __shfl_sync(0xffffffffu, pick, lstar);
}

// Warp 0: re-walk 256-entry block `bk` (its two 128-entry halves in order)
// with the arithmetic of the mass pass and return the token at the crossing.
// Both halves are loaded before the first is walked (one L2 round trip).
__device__ __forceinline__ int32_t walk_block(const float4* tp, const float4* dp, int32_t bk,
                                              int32_t nv, float2 cc, float2 ncp, float2 ncq,
                                              bool from_p, float tb, int lane) {
  const float4 ninf = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
  float4 xp[2], xq[2];
#pragma unroll
  for (int half = 0; half < 2; ++half) {
    const int32_t i = bk * 64 + half * 32 + lane;
    xp[half] = i < nv ? tp[i] : ninf;
    xq[half] = (i < nv && !from_p) ? dp[i] : xp[half];
  }
  int32_t last_pos = -1;
  float run = 0.f;
#pragma unroll
  for (int half = 0; half < 2; ++half) {
    const int32_t i = bk * 64 + half * 32 + lane;
    float hs;
    const int32_t pick = walk_half(weights4(xp[half], xq[half], cc, ncp, ncq, from_p), 4 * i,
                                   tb - run, &hs, &last_pos, lane);
    if (pick >= 0) return pick;
    run += hs;
  }
  return last_pos;  // rounding ran past the end of the block
}

template <int STRATEGY>
__global__ void __launch_bounds__(kThreads, kCtasPerSm) accept_kernel(AcceptArgs a) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  float* ring = reinterpret_cast<float*>(smem_raw);                  // [kStages][2][kChunk]
  float* block_mass = ring + kStages * 2 * kChunk;                   // [nch * 16]
  __shared__ Shared sh;
  const int32_t tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int32_t nch = (a.V + kChunk - 1) / kChunk;
  __shared__ int32_t s_early;
  if (warp == 0) {
    // mode 1: always; mode 2: when the step's frontiers leave at most half of
    // the CTAs a row (most SMs idle while the busy CTAs stream their rows)
    bool early = a.early_dependents == 1;
    if (a.early_dependents == 2 && a.cache_len != nullptr) {
      int32_t live = 0;
      for (int32_t b = lane; b < a.rows / a.D_max; b += 32)
        live += frontier_drafts(a.grid, a.cache_len[b], a.D_max);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) live += __shfl_xor_sync(0xffffffffu, live, o);
      early = 2 * live <= (int32_t)gridDim.x;
    }
    if (lane == 0) s_early = early ? 1 : 0;
  }
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&sh.full[s], 1);
      mbar_init(&sh.empty[s], kCWarps);
    }
    fence_barrier_init();
  }
  __syncthreads();
  if (s_early) pdl_launch_dependents();

  // (A) never draws and lazy (C) leaves its draws to launch_resolve: one pass
  const int32_t passes = (STRATEGY == SSD_STRATEGY_GREEDY || a.lazy) ? 1 : 2;

  // ------------------------------------------------------------ producer warp
  if (warp == kCWarps) {
    if (lane == 0) {
      uint32_t g = 0;  // chunks issued by this CTA
      for (int64_t r = blockIdx.x; r < a.rows; r += gridDim.x) {
        const int kind = row_kind(a, r);
        if (kind == 1 || kind == 2) continue;
        // the row's reference is read once: the consumers may redirect it for
        // the next round while this row's second pass is still being issued
        const float* drow =
            (a.ref_rows != nullptr && !a.ref_init) ? a.ref_rows[r] : a.drf + r * a.ld;
        for (int32_t cc = 0; cc < passes * nch; ++cc, ++g) {  // one or two passes over the row
          const int32_t ch = cc % nch;
          const int s = g % kStages;
          if (g >= kStages) mbar_wait(&sh.empty[s], ((g / kStages) - 1) & 1, a.status);
          const uint32_t bytes = (uint32_t)min(kChunk, a.V - ch * kChunk) * 4u;
          float* dst = ring + s * 2 * kChunk;
          mbar_arrive_expect_tx(&sh.full[s], 2u * bytes);
          bulk_g2s(dst, a.tgt + r * a.ld + (int64_t)ch * kChunk, bytes, &sh.full[s]);
          bulk_g2s(dst + kChunk, drow + (int64_t)ch * kChunk, bytes, &sh.full[s]);
        }
      }
    } else if (a.cache_len != nullptr) {
      // lanes 1-31: write the frontier of sequences blockIdx.x, + gridDim.x, ...
      const int32_t B = (int32_t)(a.rows / a.D_max);
      for (int32_t b = blockIdx.x; b < B; b += gridDim.x) {
        const int32_t n = frontier_drafts(a.grid, a.cache_len[b], a.D_max);
        const int32_t n_c = a.cache_len[b] - a.grid.prefix_len;
        if (lane == 1) {
          a.n_drafts_out[b] = n < 0 ? 0 : n;
          if (a.tickets != nullptr) a.tickets[b] = 0;
          if (n < 0) record_status(a.status, SSD_ERR_DEVICE_BOUNDS);
        }
        for (int32_t j = lane - 1; j < a.D_max; j += 31)
          a.draft_pos[(int64_t)b * a.D_max + j] = j < n ? n_c + j : -1;
      }
    }
    __syncwarp();
    return;
  }

  // ---------------------------------------------------------- consumer warps
  constexpr bool greedy = STRATEGY == SSD_STRATEGY_GREEDY;
  constexpr bool sample = STRATEGY == SSD_STRATEGY_SAMPLE;
  const float c = kLog2e / a.temperature;
  const float2 cc = make_float2(c, c);
  const int32_t nv = a.V >> 2;
  const int32_t nblocks = nch * kBlocksPerChunk;
  const float4 ninf = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
  uint32_t g = 0;  // chunks consumed
  for (int64_t r = blockIdx.x; r < a.rows; r += gridDim.x) {
    const int kind = row_kind(a, r);
    if (kind == 1 || kind == 2) {
      if (tid == 0) {
        a.out_tok[r] = -1;
        a.accepted[r] = 0;
        if (a.ratio) a.ratio[r] = 0.f;
        if (kind == 1 && a.lse) { a.lse[2 * r] = 0.f; a.lse[2 * r + 1] = 0.f; }
        if (kind == 2) record_status(a.status, SSD_ERR_DEVICE_BOUNDS);
        if (a.ref_rows != nullptr && a.ref_init) a.ref_rows[r] = a.drf + r * a.ld;
        if (a.lazy) a.stats[r] = make_float2(NAN, NAN);
      }
      continue;
    }
    // the bonus row draws from p alone (its draft logits are not read for it)
    const bool is_bonus = kind == 3;
    const bool row_p = sample || is_bonus;  // second pass over the weights of p
    const int32_t given_t = (a.draft_tok != nullptr && !is_bonus) ? a.draft_tok[r] : -1;
    // the row's uniforms, drawn while its first chunk is still in flight
    const float2 u = (tid == 0) ? row_uniforms(a.rng, r) : make_float2(0.f, 0.f);

    // ---- pass A: per chunk, each thread takes 8 entries of both rows
    // (float4 tid and tid + 256 of the chunk, ascending): new running maxima
    // (three-input max), one rescale per row, packed exponent arguments and
    // sums; the first argmax of q carries the p logit
    float mp = kLowest, mq = kLowest, xpa = 0.f;
    float2 sp2 = make_float2(0.f, 0.f), sq2 = sp2;
    int32_t iq = 0x7fffffff, ip = 0x7fffffff;
    for (int32_t ch = 0; ch < nch; ++ch, ++g) {
      const int s = g % kStages;
      mbar_wait(&sh.full[s], (g / kStages) & 1, a.status);
      const float4* xp4 = reinterpret_cast<const float4*>(ring + s * 2 * kChunk);
      const float4* xq4 = reinterpret_cast<const float4*>(ring + s * 2 * kChunk + kChunk);
      const int32_t cv = min(kChunk, a.V - ch * kChunk) >> 2;
      const bool in0 = tid < cv, in1 = tid + kConsumers < cv;
      const float4 p0 = in0 ? xp4[tid] : ninf, p1 = in1 ? xp4[tid + kConsumers] : ninf;
      const float4 q0 = in0 ? xq4[tid] : ninf, q1 = in1 ? xq4[tid + kConsumers] : ninf;
      const float cmp = fmax3(fmax3(p0.x, p0.y, p0.z), fmax3(p0.w, p1.x, p1.y), fmaxf(p1.z, p1.w));
      const float cmq = fmax3(fmax3(q0.x, q0.y, q0.z), fmax3(q0.w, q1.x, q1.y), fmaxf(q1.z, q1.w));
      if (greedy && cmp > mp) {  // first argmax of p (strategy A)
        const int32_t e0 = ch * kChunk + 4 * tid, e1 = e0 + 4 * kConsumers;
        if (p0.x == cmp) ip = e0;
        else if (p0.y == cmp) ip = e0 + 1;
        else if (p0.z == cmp) ip = e0 + 2;
        else if (p0.w == cmp) ip = e0 + 3;
        else if (p1.x == cmp) ip = e1;
        else if (p1.y == cmp) ip = e1 + 1;
        else if (p1.z == cmp) ip = e1 + 2;
        else ip = e1 + 3;
      }
      const float nmp = fmaxf(mp, cmp);
      if (cmq > mq) {
        const int32_t e0 = ch * kChunk + 4 * tid, e1 = e0 + 4 * kConsumers;
        if (q0.x == cmq) { iq = e0; xpa = p0.x; }
        else if (q0.y == cmq) { iq = e0 + 1; xpa = p0.y; }
        else if (q0.z == cmq) { iq = e0 + 2; xpa = p0.z; }
        else if (q0.w == cmq) { iq = e0 + 3; xpa = p0.w; }
        else if (q1.x == cmq) { iq = e1; xpa = p1.x; }
        else if (q1.y == cmq) { iq = e1 + 1; xpa = p1.y; }
        else if (q1.z == cmq) { iq = e1 + 2; xpa = p1.z; }
        else { iq = e1 + 3; xpa = p1.w; }
      }
      const float nmq = fmaxf(mq, cmq);
      // rescale of the running sums (exactly 1 when the maximum did not move;
      // the initial kLowest is finite, so no -inf - -inf)
      const float rp = ex2_approx((mp - nmp) * c), rq = ex2_approx((mq - nmq) * c);
      mp = nmp;
      mq = nmq;
      const float2 ep = exp_sum8(p0, p1, cc, make_float2(-mp * c, -mp * c));
      const float2 eq = exp_sum8(q0, q1, cc, make_float2(-mq * c, -mq * c));
      sp2 = ffma2(sp2, make_float2(rp, rp), ep);
      sq2 = ffma2(sq2, make_float2(rq, rq), eq);
      if (given_t >= 0 && (given_t / kChunk) == ch) {
        const int32_t off = given_t - ch * kChunk;  // entry inside the chunk
        const int32_t f = off >> 2, k = off & 3;
        if (f == tid || f == tid + kConsumers) {
          const float4 gp = (f == tid) ? p0 : p1, gq = (f == tid) ? q0 : q1;
          sh.xp_t = k == 0 ? gp.x : k == 1 ? gp.y : k == 2 ? gp.z : gp.w;
          sh.xq_t = k == 0 ? gq.x : k == 1 ? gq.y : k == 2 ? gq.z : gq.w;
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&sh.empty[s]);
    }
    float sp = sp2.x + sp2.y, sq = sq2.x + sq2.y;
    // the row's reference (draft) row: read here, before the barrier after
    // which this row's decision may redirect it for the next round
    const float* drow =
        (a.ref_rows != nullptr && !a.ref_init) ? a.ref_rows[r] : a.drf + r * a.ld;
    if (greedy) {  // first argmax of p over the CTA (warp tree, then the warps in order)
      float pm = mp;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const float om = __shfl_xor_sync(0xffffffffu, pm, o);
        const int32_t oi = __shfl_xor_sync(0xffffffffu, ip, o);
        if (better_arg(om, oi, pm, ip)) { pm = om; ip = oi; }
      }
      if (lane == 0) {
        sh.red_pm[warp] = pm;
        sh.red_pi[warp] = ip;
      }
    }
    // block reduction in a fixed order: xor tree in each warp, then a
    // three-level xor tree over the warps' results in warp 0
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      merge(mp, sp, __shfl_xor_sync(0xffffffffu, mp, o), __shfl_xor_sync(0xffffffffu, sp, o), c);
      const float om = __shfl_xor_sync(0xffffffffu, mq, o);
      const float os = __shfl_xor_sync(0xffffffffu, sq, o);
      const int32_t oi = __shfl_xor_sync(0xffffffffu, iq, o);
      const float op = __shfl_xor_sync(0xffffffffu, xpa, o);
      const bool take = better_arg(om, oi, mq, iq);
      merge(mq, sq, om, os, c);
      if (take) { iq = oi; xpa = op; }
    }
    if (lane == 0) {
      sh.red[warp][0] = mp;
      sh.red[warp][1] = sp;
      sh.red[warp][2] = mq;
      sh.red[warp][3] = sq;
      sh.red[warp][4] = xpa;
      sh.red_i[warp] = iq;
    }
    consumers_sync();
    if (warp == 0) {
      const bool have = lane < kCWarps;
      float Mp = have ? sh.red[lane][0] : kLowest, Sp = have ? sh.red[lane][1] : 0.f;
      float Mq = have ? sh.red[lane][2] : kLowest, Sq = have ? sh.red[lane][3] : 0.f;
      float xp_t = have ? sh.red[lane][4] : 0.f;
      int32_t t = have ? sh.red_i[lane] : 0x7fffffff;
#pragma unroll
      for (int o = kCWarps / 2; o > 0; o >>= 1) {
        merge(Mp, Sp, __shfl_xor_sync(0xffffffffu, Mp, o), __shfl_xor_sync(0xffffffffu, Sp, o), c);
        const float om = __shfl_xor_sync(0xffffffffu, Mq, o);
        const float os = __shfl_xor_sync(0xffffffffu, Sq, o);
        const int32_t oi = __shfl_xor_sync(0xffffffffu, t, o);
        const float op = __shfl_xor_sync(0xffffffffu, xp_t, o);
        const bool take = better_arg(om, oi, Mq, t);
        merge(Mq, Sq, om, os, c);
        if (take) { t = oi; xp_t = op; }
      }
      if (lane == 0 && is_bonus) {
        // the position after the last draft (horizontal stage): no draft
        // token; (A) the argmax of p, otherwise a draw from p
        const float lsp = log2f(Sp);
        if (greedy) {
          float pm = sh.red_pm[0];
          int32_t pi = sh.red_pi[0];
          for (int w = 1; w < kCWarps; ++w)
            if (better_arg(sh.red_pm[w], sh.red_pi[w], pm, pi)) { pm = sh.red_pm[w]; pi = sh.red_pi[w]; }
          a.out_tok[r] = pi;
        }
        sh.accept = greedy ? 1 : 0;
        sh.t_hat = -1;
        sh.u_res = u.y;
        sh.Cp = Mp * c + lsp;
        sh.Cq = 0.f;
        if (a.lazy) {  // drawn by launch_resolve if every draft is accepted
          a.out_tok[r] = -1;
          a.stats[r] = make_float2(sh.Cp, 0.f);
        }
        a.accepted[r] = 1;
        if (a.ratio) a.ratio[r] = 0.f;
        if (a.lse) {
          a.lse[2 * r] = Mp / a.temperature + lsp * kLn2;
          a.lse[2 * r + 1] = 0.f;
        }
      } else if (lane == 0) {
        float xq_t = Mq;
        if (given_t >= 0) {
          t = given_t;
          xp_t = sh.xp_t;
          xq_t = sh.xq_t;
        }
        const bool valid_t = t >= 0 && t < a.V;
        const float lsp = log2f(Sp), lsq = log2f(Sq);
        float ratio = 0.f;
        bool acc = false;
        if (valid_t) {
          const float l2p = (xp_t - Mp) * c - lsp;
          const float l2q = (xq_t - Mq) * c - lsq;
          ratio = exp2f(l2p - l2q);
          acc = u.x < fminf(ratio, 1.0f);
        } else {
          record_status(a.status, SSD_ERR_DEVICE_BOUNDS);  // non-finite logits
        }
        int32_t out = acc ? t : -1;
        if (greedy && valid_t) {  // (A): the first argmax of p over the warps, in order
          float pm = sh.red_pm[0];
          int32_t pi = sh.red_pi[0];
          for (int w = 1; w < kCWarps; ++w)
            if (better_arg(sh.red_pm[w], sh.red_pi[w], pm, pi)) { pm = sh.red_pm[w]; pi = sh.red_pi[w]; }
          out = pi;
          acc = pi == t;
        }
        // (C) draws on rejection, (B) always; (A) never
        sh.accept = !valid_t ? 2 : (sample ? 0 : (greedy || acc) ? 1 : 0);
        sh.t_hat = t;
        sh.u_res = u.y;
        sh.Cp = Mp * c + lsp;
        sh.Cq = Mq * c + lsq;
        // round 1 starts every reference at the draft row; a draw that differs
        // from the token redirects it below (sampling) or here (the others)
        if (sample && a.ref_rows != nullptr && a.ref_init) a.ref_rows[r] = drow;
        if (!sample) {
          a.accepted[r] = acc ? 1 : 0;
          if (acc || greedy) a.out_tok[r] = out;
          // the next round's reference of a row this round did not accept
          if (a.ref_rows != nullptr && valid_t && !acc) a.ref_rows[r] = a.tgt + r * a.ld;
          else if (a.ref_rows != nullptr && a.ref_init) a.ref_rows[r] = drow;
        }
        if (!valid_t) {
          a.accepted[r] = 0;
          a.out_tok[r] = -1;
        }
        if (a.lazy) {  // a rejected row's token is drawn by launch_resolve if committed
          if (sh.accept == 0) a.out_tok[r] = -1;
          a.stats[r] = valid_t ? make_float2(sh.Cp, sh.Cq) : make_float2(NAN, NAN);
        }
        if (a.ratio) a.ratio[r] = ratio;
        if (a.lse) {
          a.lse[2 * r] = Mp / a.temperature + lsp * kLn2;
          a.lse[2 * r + 1] = Mq / a.temperature + lsq * kLn2;
        }
      }
    }
    consumers_sync();
    if (passes == 1) continue;  // uniform; sh is rewritten only after the next row's pass A
    const bool draw = (sh.accept == 0);
    const float2 ncp = make_float2(-sh.Cp, -sh.Cp), ncq = make_float2(-sh.Cq, -sh.Cq);

    // ---- pass B: second-pass chunks; residual mass of every 256-entry block
    for (int32_t ch = 0; ch < nch; ++ch, ++g) {
      const int s = g % kStages;
      mbar_wait(&sh.full[s], (g / kStages) & 1, a.status);
      if (draw) {
        const float4* xp4 = reinterpret_cast<const float4*>(ring + s * 2 * kChunk);
        const float4* xq4 = reinterpret_cast<const float4*>(ring + s * 2 * kChunk + kChunk);
        const int32_t cv = min(kChunk, a.V - ch * kChunk) >> 2;
        const int32_t i0 = warp * 64 + lane, i1 = i0 + 32;
        float4 w0 = make_float4(0.f, 0.f, 0.f, 0.f), w1 = w0;
        if (i0 < cv) w0 = weights4(xp4[i0], xq4[i0], cc, ncp, ncq, row_p);
        if (i1 < cv) w1 = weights4(xp4[i1], xq4[i1], cc, ncp, ncq, row_p);
        const float m = warp_sum(((w0.x + w0.y) + (w0.z + w0.w)) + ((w1.x + w1.y) + (w1.z + w1.w)));
        if (lane == 0) block_mass[ch * kBlocksPerChunk + warp] = m;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&sh.empty[s]);
    }
    if (!draw) continue;  // uniform
    consumers_sync();
    const float4* tp = reinterpret_cast<const float4*>(a.tgt + r * a.ld);
    const float4* dp = reinterpret_cast<const float4*>(drow);
    if (warp == 0) {
      float tb;
      int32_t bk = find_block(block_mass, nblocks, sh.u_res, &tb, lane);
      bool from_p = row_p;
      if (bk < 0 && !row_p) {
        // zero residual mass: the same draw from p (block masses of p itself)
        from_p = true;
        for (int32_t b0 = 0; b0 < nblocks; ++b0) {
          const int32_t i0 = b0 * 64 + lane, i1 = i0 + 32;
          float4 w0 = make_float4(0.f, 0.f, 0.f, 0.f), w1 = w0;
          if (i0 < nv) w0 = weights4(tp[i0], tp[i0], cc, ncp, ncq, true);
          if (i1 < nv) w1 = weights4(tp[i1], tp[i1], cc, ncp, ncq, true);
          const float m = warp_sum(((w0.x + w0.y) + (w0.z + w0.w)) + ((w1.x + w1.y) + (w1.z + w1.w)));
          if (lane == 0) block_mass[b0] = m;
        }
        __syncwarp();
        bk = find_block(block_mass, nblocks, sh.u_res, &tb, lane);
      }
      if (bk < 0) {
        if (lane == 0) {  // no positive mass at all (non-finite logits)
          a.out_tok[r] = -1;
          if (sample || is_bonus) a.accepted[r] = 0;
          record_status(a.status, SSD_ERR_DEVICE_BOUNDS);
        }
      } else if (dbg_in(bk, nblocks, a.status)) {
        const int32_t pick = walk_block(tp, dp, bk, nv, cc, ncp, ncq, from_p, tb, lane);
        if (lane == 0) {
          a.out_tok[r] = pick;
          if (sample && !is_bonus) {
            a.accepted[r] = pick == sh.t_hat ? 1 : 0;
            if (a.ref_rows != nullptr && pick != sh.t_hat) a.ref_rows[r] = a.tgt + r * a.ld;
            else if (a.ref_rows != nullptr && a.ref_init) a.ref_rows[r] = drow;
          }
        }
      }
    }
    consumers_sync();  // block masses and sh are reused by the next row
  }
}

// After a lazy acceptance pass: the counts and the one committed draw per
// sequence.  Grid (parts, B), one warp per CTA, so that the CTAs fit in the
// registers an attention kernel leaves free on an SM and run beside it.
// Every CTA of sequence b takes the counts' leading run (part 0 writes the
// counts); if they commit a drawn token — the residual token of the first
// rejected draft, or the bonus token after a fully accepted horizontal
// frontier — part k computes the residual masses of 256-entry blocks
// [kRBlocks k, kRBlocks (k + 1)) with the arithmetic of pass B (same lane
// layout, weights and warp sums, so every block mass is bit-identical) into
// global memory; the last part to finish (a ticket per sequence) scans the
// masses in vocabulary order and re-walks the chosen block exactly as the
// eager kernel does for that row.
constexpr int kRBlocks = 2;  // blocks per part: one batch of loads

__device__ __forceinline__ void resolve_part_masses(const float4* tp, const float4* dp, int32_t bk0,
                                                    int32_t bk1, int32_t nv, float2 cc, float2 ncp,
                                                    float2 ncq, bool from_p, float* mass, int lane) {
  for (int32_t b0 = bk0; b0 < bk1; b0 += 2) {
    float4 xp[2][2], xq[2][2];
#pragma unroll
    for (int k = 0; k < 2; ++k) {
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        const int32_t i = (b0 + k) * 64 + half * 32 + lane;
        const bool in = b0 + k < bk1 && i < nv;
        xp[k][half] = in ? tp[i] : make_float4(0.f, 0.f, 0.f, 0.f);
        xq[k][half] = (in && !from_p) ? dp[i] : xp[k][half];
      }
    }
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      const int32_t bk = b0 + k;
      if (bk >= bk1) break;  // warp-uniform
      float4 w0 = make_float4(0.f, 0.f, 0.f, 0.f), w1 = w0;
      if (bk * 64 + lane < nv) w0 = weights4(xp[k][0], xq[k][0], cc, ncp, ncq, from_p);
      if (bk * 64 + 32 + lane < nv) w1 = weights4(xp[k][1], xq[k][1], cc, ncp, ncq, from_p);
      const float m = warp_sum(((w0.x + w0.y) + (w0.z + w0.w)) + ((w1.x + w1.y) + (w1.z + w1.w)));
      if (lane == 0) mass[bk] = m;
    }
  }
}

__global__ void __launch_bounds__(32, 32) resolve_kernel(ResolveArgs a) {
  extern __shared__ __align__(16) float rmass[];  // [nblocks], last part only
  const int32_t part = blockIdx.x, b = blockIdx.y, lane = threadIdx.x;
  const int32_t nblocks = ((a.V + kChunk - 1) / kChunk) * kBlocksPerChunk;  // resolve_blocks(V)
  const int32_t nv = a.V >> 2;
  const int32_t bk0 = part * kRBlocks, bk1 = min(nblocks, bk0 + kRBlocks);
  // The first draft is the most likely committed rejection: its statistics and
  // this part's blocks of both rows are loaded before the counts are known.
  const int64_t r0 = (int64_t)b * a.D_max;
  const float2 st0 = a.stats[r0];
  float4 xp[kRBlocks][2], xq[kRBlocks][2];
  auto load_part = [&](const float4* tp, const float4* dp, bool from_p) {
#pragma unroll
    for (int k = 0; k < kRBlocks; ++k)
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        const int32_t i = (bk0 + k) * 64 + half * 32 + lane;
        const bool in = bk0 + k < bk1 && i < nv;
        xp[k][half] = in ? tp[i] : make_float4(0.f, 0.f, 0.f, 0.f);
        xq[k][half] = (in && !from_p) ? dp[i] : xp[k][half];
      }
  };
  load_part(reinterpret_cast<const float4*>(a.tgt + r0 * a.ld),
            reinterpret_cast<const float4*>(a.drf + r0 * a.ld), false);
  int32_t n = a.n_drafts[b];
  const bool bad_n = n < 0 || n > a.D_max;  // a caller's frontier (ssd_verify_accept)
  n = bad_n ? (n < 0 ? 0 : a.D_max) : n;
  if (part == 0 && bad_n && lane == 0) record_status(a.status, SSD_ERR_DEVICE_BOUNDS);
  const int32_t prefix = sequence_counts(a.grid, a.commit, b, a.D_max, a.cache_len, n, a.accepted,
                                         a.accepted_count, a.accepted_prefix, a.next_cache_len,
                                         lane, part == 0);
  int32_t j = -1;
  if (n > 0 && prefix < n) j = prefix;                             // first rejected draft
  else if (a.bonus && n > 0 && prefix == n && n < a.D_max) j = n;  // the bonus row
  const int64_t r = r0 + (j < 0 ? 0 : j);
  // (debug builds: the committed row against the batch's rows)
  if (!dbg_in(r, (int64_t)a.B * a.D_max, a.status)) {
    if (pdl_first_block()) pdl_wait();
    return;
  }
  const float2 st = j < 0 ? make_float2(NAN, NAN) : (j == 0 ? st0 : a.stats[r]);
  if (!(st.x == st.x)) {  // nothing to draw, or an invalid row the acceptance pass reported
    if (pdl_first_block()) pdl_wait();
    return;
  }
  const bool is_bonus = j == n;
  const float c = kLog2e / a.temperature;
  const float2 cc = make_float2(c, c);
  const float2 ncp = make_float2(-st.x, -st.x), ncq = make_float2(-st.y, -st.y);
  const float4* tp = reinterpret_cast<const float4*>(a.tgt + r * a.ld);
  const float4* dp = reinterpret_cast<const float4*>(a.drf + r * a.ld);
  float* gmass = a.mass + (int64_t)b * nblocks;
  if (j != 0) load_part(tp, dp, is_bonus);  // the speculative rows were not the committed one
  // this part's block masses, with the arithmetic of resolve_part_masses
#pragma unroll
  for (int k = 0; k < kRBlocks; ++k) {
    const int32_t bk = bk0 + k;
    if (bk >= bk1) break;  // warp-uniform
    float4 w0 = make_float4(0.f, 0.f, 0.f, 0.f), w1 = w0;
    if (bk * 64 + lane < nv) w0 = weights4(xp[k][0], xq[k][0], cc, ncp, ncq, is_bonus);
    if (bk * 64 + 32 + lane < nv) w1 = weights4(xp[k][1], xq[k][1], cc, ncp, ncq, is_bonus);
    const float m = warp_sum(((w0.x + w0.y) + (w0.z + w0.w)) + ((w1.x + w1.y) + (w1.z + w1.w)));
    if (lane == 0) gmass[bk] = m;
  }
  // last part to finish: its fence orders every part's masses before its ticket
  __threadfence();
  int32_t last = 0;
  if (lane == 0) last = atomicAdd(&a.tickets[b], 1) == (int32_t)gridDim.x - 1;
  last = __shfl_sync(0xffffffffu, last, 0);
  if (!last) {
    if (pdl_first_block()) pdl_wait();
    return;
  }
  __threadfence();
  for (int32_t k = lane; k < nblocks; k += 32) rmass[k] = __ldcg(gmass + k);
  __syncwarp();
  const float u_res = row_uniforms(a.rng, r).y;
  float tb = 0.f;
  int32_t bk = find_block(rmass, nblocks, u_res, &tb, lane);
  bool from_p = is_bonus;
  if (bk < 0 && !is_bonus) {
    // zero residual mass: the same draw from p (block masses of p itself)
    from_p = true;
    __syncwarp();
    resolve_part_masses(tp, tp, 0, nblocks, nv, cc, ncp, ncq, true, rmass, lane);
    __syncwarp();
    bk = find_block(rmass, nblocks, u_res, &tb, lane);
  }
  if (bk < 0) {
    if (lane == 0) {  // no positive mass at all (non-finite logits)
      a.out_tok[r] = -1;
      if (is_bonus) a.accepted[r] = 0;
      record_status(a.status, SSD_ERR_DEVICE_BOUNDS);
    }
  } else if (dbg_in(bk, nblocks, a.status)) {
    const int32_t pick = walk_block(tp, dp, bk, nv, cc, ncp, ncq, from_p, tb, lane);
    if (lane == 0) a.out_tok[r] = pick;
  }
  // Under a programmatic launch after the attention (the step's schedule; the
  // acceptance pass completed before the attention let this kernel in): block
  // 0 exits only after the attention, so that stream order holds.
  if (pdl_first_block()) pdl_wait();
}

}  // namespace

bool accept_supported(int32_t V) { return V <= kMaxV; }

cudaError_t launch_accept(const AcceptArgs& a, cudaStream_t stream) {
  if (a.rows == 0) return cudaSuccess;
  const int32_t nch = (a.V + kChunk - 1) / kChunk;
  const size_t smem = (size_t)kStages * 2 * kChunk * sizeof(float) +
                      (size_t)nch * kBlocksPerChunk * sizeof(float);
  const int64_t grid = std::min<int64_t>(a.rows, (int64_t)kCtasPerSm * device_sm_count());
  auto launch = [&](auto kernel) {
    cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    kernel<<<(unsigned)grid, kThreads, smem, stream>>>(a);
    return cudaGetLastError();
  };
  switch (a.strategy) {
    case SSD_STRATEGY_GREEDY: return launch(accept_kernel<SSD_STRATEGY_GREEDY>);
    case SSD_STRATEGY_SAMPLE: return launch(accept_kernel<SSD_STRATEGY_SAMPLE>);
    default: return launch(accept_kernel<SSD_STRATEGY_ACCEPT_REJECT>);
  }
}

int32_t resolve_blocks(int32_t V) { return ((V + kChunk - 1) / kChunk) * kBlocksPerChunk; }

cudaError_t launch_resolve(const ResolveArgs& a, bool pdl, cudaStream_t stream) {
  if (a.B == 0) return cudaSuccess;
  const int32_t nblocks = resolve_blocks(a.V);
  const size_t smem = (size_t)nblocks * sizeof(float);
  cudaError_t e = cudaFuncSetAttribute(resolve_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  const dim3 grid((unsigned)((nblocks + kRBlocks - 1) / kRBlocks), (unsigned)a.B);
  return launch_kernel(resolve_kernel, grid, dim3(32), smem, stream, pdl, a);
}

}  // namespace ssd
