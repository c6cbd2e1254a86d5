// lmhead.cu — fused lm_head + acceptance (step a6).  Sec. 3.3, after Eq. 2:
// draft tokens are decoded through the base model's GenHead, a linear map
// from the (normalised) hidden state to vocabulary logits.  Verification
// needs it for the target hidden states H_t and the draft hidden states H_d:
//   l_p = H_t W_t,  l_q = H_d W_d   ([rows x K] x [K x V])
// followed by strategy (C) of Sec. 3.3 on every row (accept with probability
// min(p/q, 1), otherwise draw from [p - q]_+), exactly as accept.cu, but
// with the logits never written to memory.
//
// Design (GB300, tcgen05 + TMEM):
//  * one CTA per tile of 128 vocabulary entries; draft rows on the MMA's M
//    dimension (TMEM lanes, padded to 128 per row tile), vocabulary on N, so
//    each epilogue thread owns one row's 128 logits of the tile;
//  * A = hidden states (K-major), B = weights (MN-major: the vocabulary is
//    contiguous in W[K][V]); both staged by TMA with the 128-byte swizzle
//    through a 3-stage mbarrier ring, two threads producing (hidden states;
//    weights, one copy per tile through a 3D view), one thread
//    issuing tcgen05.mma (bf16 x bf16 -> fp32) into two TMEM accumulators
//    (target, draft), tcgen05.commit releasing each stage;
//  * epilogue: tcgen05.ld of each row's tile, per-tile softmax partials to a
//    small workspace, a bounded grid barrier (the launch is cooperative, so
//    every CTA is resident), a warp-parallel combine of each row's partials
//    in a fixed order by one CTA (row r by CTA r mod the grid), which takes
//    the decision and publishes the row's normalisers; a second barrier; the
//    rows to draw (every rejected row, or, inside a one-round prefix-commit
//    step, only each sequence's first rejection: the one token the commit
//    keeps), their per-tile residual masses, a third barrier, and the CTA
//    holding the CDF crossing scans its row tile sequentially.  Logits stay
//    in TMEM throughout.
#include "kernels.cuh"

namespace ssd {

namespace {

constexpr int kBM = 128;        // rows per MMA tile (TMEM lanes)
constexpr int kBN = 128;        // vocabulary entries per CTA
constexpr int kBK = 64;         // K per stage: one 128-byte swizzle atom of bf16
constexpr int kMMAK = 16;       // K per tcgen05.mma (kind::f16)
constexpr int kThreadsL = 512;  // warps 0-3 own the 128 TMEM lanes; all 16 share the combines
constexpr int kTmemWarps = 4;
constexpr int kCombWarps = kThreadsL / 32;
constexpr int kMaxTilesPerLane = 8;  // vocabulary tiles per lane in the combines: V <= 32768
constexpr int kMaxRowTiles = 2; // rows <= 256
constexpr float kLog2eL = 1.4426950408889634f;
constexpr float kLn2L = 0.6931471805599453f;

constexpr int kTileA = kBM * kBK * 2;   // 16 KB: [128 rows x 64 K] bf16
constexpr int kTileB = kBK * kBN * 2;   // 16 KB: [64 K x 128 vocab] bf16 (two 64-wide boxes)

struct LmPartial {  // one row, one vocabulary tile (32 bytes)
  float max_p, sum_p, max_q, sum_q;
  float xq_c, xp_c;  // logits at the tile's candidate (argmax of q, or the given token)
  int32_t cand;      // candidate index, -1 if none
  float pad;
};

// Instruction descriptor, kind::f16: fp32 D, bf16 A and B, A K-major,
// B MN-major, N = 128, M = 128.
constexpr uint32_t kIdesc = idesc_bf16(kBM, kBN, false, true);

__device__ __forceinline__ bool better(float v, int32_t i, float bv, int32_t bi) {
  return v > bv || (v == bv && (uint32_t)i < (uint32_t)bi);
}

__device__ __forceinline__ void merge_ms(float& m, float& s, float m2, float s2, float c) {
  const float mn = fmaxf(m, m2);
  if (mn == -INFINITY) return;
  s = s * ex2_approx((m - mn) * c) + s2 * ex2_approx((m2 - mn) * c);
  m = mn;
}

__device__ __forceinline__ uint32_t ld_acquire(const unsigned int* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Bounded grid barrier over `ncta` co-resident CTAs (cooperative launch).
// ctr[0] counts arrivals over the kernel's barriers (cumulative targets);
// ctr[1] is an abort flag: a CTA that gives up waiting (after max_polls polls,
// SSD_ERR_TIMEOUT recorded) raises it before it arrives anywhere else, so a
// slower CTA that later sees the count reached through that CTA's next
// arrival fails too instead of going on with missing partials.  Returns false
// in every thread if this CTA gave up or the kernel was aborted.
__device__ bool grid_barrier(unsigned int* ctr, unsigned int target, int32_t* status,
                             int32_t* flag, uint32_t max_polls) {
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    atomicAdd(ctr, 1u);
    bool ok = false;
    for (uint32_t i = 0; i < max_polls; ++i) {
      if (ld_acquire(ctr) >= target) { ok = true; break; }
      if (i > 256) __nanosleep(64);
    }
    if (ok) {
      ok = ld_acquire(ctr + 1) == 0u;
    } else {
      atomicExch(ctr + 1, 1u);
      record_status(status, SSD_ERR_TIMEOUT);
    }
    __threadfence();
    *flag = ok ? 1 : 0;
  }
  __syncthreads();
  return *flag != 0;
}

struct LmSmemRow {  // per-row results of the decision, broadcast inside the CTA
  float Cp, Cq;     // log2-domain normalisers max * c + log2(sum)
  float u_res;
  int32_t state;    // 0 skip (padding / accepted / invalid), 1 rejected: draw
  int32_t cstar;    // CTA holding the crossing for this row, -1 none
  float tc;         // remaining target inside that CTA's tile (INF: last positive)
  int32_t from_p;   // 1: zero residual mass, draw from p
  int32_t pad;
};

struct LmRowRec {   // one row's combine, for every CTA after the second barrier
  float Cp, Cq, u_res;
  int32_t state;    // 1: valid and rejected (a draw candidate), else 0
};

struct LmLaunch {
  int32_t ncta, mt, stages;
  LmPartial* part;      // [rows][ncta]
  float* mass;          // [rows][ncta]
  LmRowRec* rec;        // [rows] each row's decision, written by the CTA that combined it
  unsigned int* barrier;
  uint32_t max_polls;   // limit of every bounded wait of the kernel
  uint32_t shortfall;   // extra arrivals each grid barrier waits for (0; > 0 in tests)
};

__global__ void __launch_bounds__(kThreadsL, 1)
lmhead_accept_kernel(const __grid_constant__ CUtensorMap tmHt, const __grid_constant__ CUtensorMap tmHd,
                     const __grid_constant__ CUtensorMap tmWt, const __grid_constant__ CUtensorMap tmWd,
                     LmHeadArgs a, LmLaunch L) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int mt = L.mt, S = L.stages;
  const int stage_bytes = 2 * mt * kTileA + 2 * kTileB;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S * stage_bytes);
  uint64_t* empty = full + S;
  uint64_t* done = empty + S;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
  int32_t* flag = reinterpret_cast<int32_t*>(tmem_slot + 1);
  int32_t* fail = flag + 1;
  LmSmemRow* rowinfo = reinterpret_cast<LmSmemRow*>(fail + 2);  // [mt * 128]

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int cta = blockIdx.x;
  const int32_t v0 = cta * kBN;
  const int32_t nkb = a.K / kBK;
  const uint32_t ncols = (uint32_t)(mt * 2 * kBN);  // target + draft accumulators per row tile

  // ---- set-up: barriers, TMEM
  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(done, 1);
    *fail = 0;
    fence_barrier_init();
  }
  if (warp == 0) {
    tmem_alloc(tmem_slot, ncols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  // ---- main loop: warp 0 lane 0 produces, warp 1 lane 0 issues the MMAs.
  // The other lanes of those two warps park at __syncwarp: spinning on an
  // mbarrier in the same warp would let a suspended try_wait of theirs hold
  // up the lane that drives the pipeline.
  if (warp == 0) {
    // Lane 0 issues the hidden-state tiles, lane 1 the two weight tiles (one
    // copy each through the 3D view {64, K, V / 64}): one thread issues only a
    // few million copies per second.
    if (lane < 2) {
    const uint64_t pol = policy_evict_first();     // weights: read once
    const uint64_t pol_h = policy_evict_last();    // hidden states: read by every CTA
    const uint32_t bytes = (uint32_t)stage_bytes;
    for (int kb = 0; kb < nkb; ++kb) {
      const int s = kb % S;
      int stop = 0;
      if (lane == 0) {
        if (kb >= S && !mbar_wait(&empty[s], ((kb / S) - 1) & 1, a.status, L.max_polls)) {
          *fail = 1;
          stop = 1;
        } else {
          mbar_arrive_expect_tx(&full[s], bytes);
        }
      }
      stop = __shfl_sync(0x3u, stop, 0);  // the stage is free and its bytes expected
      if (stop) break;
      unsigned char* st = smem + s * stage_bytes;
      if (lane == 0) {
        for (int m = 0; m < mt; ++m) {
          tma_load_2d(st + m * kTileA, &tmHt, kb * kBK, m * kBM, &full[s], pol_h);
          tma_load_2d(st + (mt + m) * kTileA, &tmHd, kb * kBK, m * kBM, &full[s], pol_h);
        }
      } else {
        unsigned char* bt = st + 2 * mt * kTileA;
        tma_load_3d(bt, &tmWt, 0, kb * kBK, v0 / 64, &full[s], pol);
        tma_load_3d(bt + kTileB, &tmWd, 0, kb * kBK, v0 / 64, &full[s], pol);
      }
    }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
    for (int kb = 0; kb < nkb; ++kb) {
      const int s = kb % S;
      if (!mbar_wait(&full[s], (kb / S) & 1, a.status, L.max_polls)) { *fail = 1; break; }
      tc_fence_after();
      const uint32_t st = smem_u32(smem + s * stage_bytes);
      const uint32_t bt = st + 2 * mt * kTileA, bd = bt + kTileB;
#pragma unroll
      for (int kk = 0; kk < kBK / kMMAK; ++kk) {
        // B (MN-major): 64-wide vocabulary atoms 8 KB apart (LBO), 8-row K groups
        // 1 KB apart (SBO); one MMA's K = 16 rows = 2 KB further per step.
        const uint64_t db_t = smem_desc(bt + kk * 2048, 8192, 1024);
        const uint64_t db_d = smem_desc(bd + kk * 2048, 8192, 1024);
        for (int m = 0; m < mt; ++m) {
          // A (K-major): 8-row groups 1 KB apart (SBO); K = 16 is 32 bytes along the row.
          const uint64_t da_t = smem_desc(st + m * kTileA + kk * 32, 16, 1024);
          const uint64_t da_d = smem_desc(st + (mt + m) * kTileA + kk * 32, 16, 1024);
          const uint32_t acc = (kb > 0 || kk > 0) ? 1u : 0u;
          mma_ss(tmem + m * 2 * kBN, da_t, db_t, kIdesc, acc);
          mma_ss(tmem + m * 2 * kBN + kBN, da_d, db_d, kIdesc, acc);
        }
      }
      mma_commit(&empty[s]);
    }
    mma_commit(done);
    }
    __syncwarp();
  }
  // every thread waits for the accumulators
  const bool mma_ok = mbar_wait(done, 0, a.status, L.max_polls);
  tc_fence_after();
  bool ok = __syncthreads_and(mma_ok) != 0;
  ok = ok && (*fail == 0);

  const float c = kLog2eL / a.temperature;
  const int32_t rows = a.rows;
  // TMEM lane quarter of this warp: lanes 32*warp .. +31 (row tile m, row m*128 + tid)
  const uint32_t lane_off = (uint32_t)(warp * 32) << 16;

  // ---- epilogue 1: per-tile softmax partials of every row (TMEM warps)
  for (int m = 0; m < mt && ok && warp < kTmemWarps; ++m) {
    const int32_t row = m * kBM + tid;
    const uint32_t tp = tmem + lane_off + m * 2 * kBN, tq = tp + kBN;
    float mp = -INFINITY, sp = 0.f, mq = -INFINITY, sq = 0.f;
    float xq_c = -INFINITY, xp_c = 0.f;
    int32_t cand = -1;
    const int32_t given = (a.draft_tok != nullptr && row < rows) ? a.draft_tok[row] : -1;
    float v[32], w[32];
#pragma unroll 1
    for (int ch = 0; ch < kBN / 32; ++ch) {
      tmem_ld32(tp + ch * 32, v);
      tmem_ld32(tq + ch * 32, w);
      float cmp = -INFINITY, cmq = -INFINITY;
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        cmp = fmaxf(cmp, v[i]);
        cmq = fmaxf(cmq, w[i]);
      }
      if (given < 0 && cmq > xq_c) {  // first maximum of q (ascending scan)
#pragma unroll
        for (int i = 31; i >= 0; --i)
          if (w[i] == cmq) { cand = v0 + ch * 32 + i; xp_c = v[i]; }
        xq_c = cmq;
      }
      if (given >= v0 + ch * 32 && given < v0 + ch * 32 + 32) {
#pragma unroll
        for (int i = 0; i < 32; ++i)
          if (given == v0 + ch * 32 + i) { cand = given; xp_c = v[i]; xq_c = w[i]; }
      }
      float lp = 0.f, lq = 0.f;
      const float cmpc = cmp * c, cmqc = cmq * c;
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        lp += ex2_approx(fmaf(v[i], c, -cmpc));
        lq += ex2_approx(fmaf(w[i], c, -cmqc));
      }
      merge_ms(mp, sp, cmp, lp, c);
      merge_ms(mq, sq, cmq, lq, c);
    }
    if (row < rows) {
      LmPartial P;
      P.max_p = mp;
      P.sum_p = sp;
      P.max_q = mq;
      P.sum_q = sq;
      P.xq_c = cand >= 0 ? xq_c : -INFINITY;
      P.xp_c = xp_c;
      P.cand = cand;
      P.pad = 0.f;
      reinterpret_cast<float4*>(L.part + (int64_t)row * L.ncta + cta)[0] =
          make_float4(P.max_p, P.sum_p, P.max_q, P.sum_q);
      reinterpret_cast<float4*>(L.part + (int64_t)row * L.ncta + cta)[1] =
          make_float4(P.xq_c, P.xp_c, __int_as_float(P.cand), 0.f);
    }
  }
  ok = grid_barrier(L.barrier, (unsigned)L.ncta + L.shortfall, a.status, flag, L.max_polls) && ok;

  // ---- epilogue 2: combine the partials of each row and decide.  Row r is
  // combined by CTA r % ncta alone (one warp per row; lane l merges tiles l,
  // l + 32, ... in order, then a xor tree), which writes its outputs and its
  // record for the other CTAs.  All loads of a row are issued before any merge.
  for (int32_t row = cta + L.ncta * warp; row < rows && ok; row += L.ncta * kCombWarps) {
    bool pad = false;
    if (a.n_drafts != nullptr) {
      const int32_t b = row / a.D_max, j = row - b * a.D_max;
      pad = j >= a.n_drafts[b];
    }
    if (pad) {
      if (lane == 0) {
        L.rec[row].state = 0;
        a.out_tok[row] = -1;
        a.accepted[row] = 0;
        if (a.ratio) a.ratio[row] = 0.f;
        if (a.lse) { a.lse[2 * row] = 0.f; a.lse[2 * row + 1] = 0.f; }
      }
      continue;
    }
    const float4* prow = reinterpret_cast<const float4*>(L.part + (int64_t)row * L.ncta);
    float4 q0[kMaxTilesPerLane], q1[kMaxTilesPerLane];
#pragma unroll
    for (int j = 0; j < kMaxTilesPerLane; ++j) {
      const int k = lane + 32 * j;
      if (k < L.ncta) {
        q0[j] = __ldcg(prow + 2 * k);
        q1[j] = __ldcg(prow + 2 * k + 1);
      }
    }
    float Mp = -INFINITY, Sp = 0.f, Mq = -INFINITY, Sq = 0.f, xq = -INFINITY, xp = 0.f;
    int32_t t = 0x7fffffff;
#pragma unroll
    for (int j = 0; j < kMaxTilesPerLane; ++j) {
      if (lane + 32 * j < L.ncta) {
        merge_ms(Mp, Sp, q0[j].x, q0[j].y, c);
        merge_ms(Mq, Sq, q0[j].z, q0[j].w, c);
        const int32_t ck = __float_as_int(q1[j].z);
        if (ck >= 0 && better(q1[j].x, ck, xq, t)) { xq = q1[j].x; xp = q1[j].y; t = ck; }
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      merge_ms(Mp, Sp, __shfl_xor_sync(0xffffffffu, Mp, o), __shfl_xor_sync(0xffffffffu, Sp, o), c);
      merge_ms(Mq, Sq, __shfl_xor_sync(0xffffffffu, Mq, o), __shfl_xor_sync(0xffffffffu, Sq, o), c);
      const float oq = __shfl_xor_sync(0xffffffffu, xq, o);
      const float op = __shfl_xor_sync(0xffffffffu, xp, o);
      const int32_t ot = __shfl_xor_sync(0xffffffffu, t, o);
      if (better(oq, ot, xq, t)) { xq = oq; xp = op; t = ot; }
    }
    if (lane == 0) {
      const int32_t given = a.draft_tok != nullptr ? a.draft_tok[row] : -1;
      const bool valid_t = (t >= 0 && t < a.V) && (given < 0 || t == given);
      float ratio = 0.f;
      bool acc = false;
      const float2 u = row_uniforms(a.rng, row);
      if (valid_t) {
        const float l2p = (xp - Mp) * c - log2f(Sp);
        const float l2q = (xq - Mq) * c - log2f(Sq);
        ratio = exp2f(l2p - l2q);
        acc = u.x < fminf(ratio, 1.0f);
      }
      LmRowRec rr;
      rr.Cp = Mp * c + log2f(Sp);
      rr.Cq = Mq * c + log2f(Sq);
      rr.u_res = u.y;
      rr.state = (valid_t && !acc) ? 1 : 0;
      L.rec[row] = rr;
      if (!valid_t) record_status(a.status, SSD_ERR_DEVICE_BOUNDS);
      a.accepted[row] = acc ? 1 : 0;
      if (acc) a.out_tok[row] = t;
      else a.out_tok[row] = -1;  // a drawn row's token is written in epilogue 5
      if (a.ratio) a.ratio[row] = ratio;
      if (a.lse) {
        a.lse[2 * row] = Mp / a.temperature + log2f(Sp) * kLn2L;
        a.lse[2 * row + 1] = Mq / a.temperature + log2f(Sq) * kLn2L;
      }
    }
  }
  ok = grid_barrier(L.barrier, 2u * ((unsigned)L.ncta + L.shortfall), a.status, flag,
                    L.max_polls) && ok;

  // ---- the rows to draw, in every CTA: every valid rejected row, or (lazy)
  // the first rejected row of each sequence among its drafts
  int32_t* first = reinterpret_cast<int32_t*>(rowinfo + mt * kBM);  // [rows / D_max]
  const bool lazy = a.lazy != 0 && a.n_drafts != nullptr;
  const int32_t ngroups = lazy ? rows / a.D_max : 0;
  for (int32_t g = tid; g < ngroups; g += kThreadsL) first[g] = 0x7fffffff;
  __syncthreads();
  if (lazy && ok) {
    for (int32_t row = tid; row < rows; row += kThreadsL) {
      const int32_t b = row / a.D_max, j = row - b * a.D_max;
      if (j < a.n_drafts[b] && __ldcg(a.accepted + row) == 0) atomicMin(&first[b], j);
    }
  }
  __syncthreads();
  for (int32_t r = tid; r < mt * kBM; r += kThreadsL) {
    LmSmemRow& ri = rowinfo[r];
    ri.state = 0;
    ri.from_p = 0;
    ri.cstar = -1;
    if (r < rows && ok) {
      // the record of another CTA, read from L2
      const float4 rv = __ldcg(reinterpret_cast<const float4*>(L.rec + r));
      const bool pick = __float_as_int(rv.w) == 1 &&
                        (!lazy || r - (r / a.D_max) * a.D_max == first[r / a.D_max]);
      if (pick) {
        ri.Cp = rv.x;
        ri.Cq = rv.y;
        ri.u_res = rv.z;
        ri.state = 1;
      }
    }
  }
  __syncthreads();

  // ---- epilogue 3: residual mass of this tile for every row to draw
  // (sequential over the tile in vocabulary order; TMEM warps)
  for (int m = 0; m < mt && ok && warp < kTmemWarps; ++m) {
    const int32_t row = m * kBM + tid;
    const LmSmemRow& ri = rowinfo[m * kBM + tid];
    const uint32_t tp = tmem + lane_off + m * 2 * kBN, tq = tp + kBN;
    float mass = 0.f;
    float v[32], w[32];
    // every lane of the warp takes part in tcgen05.ld; rows that do not draw
    // simply discard the values
    const bool draw = row < rows && ri.state == 1;
    if (!__any_sync(0xffffffffu, draw)) continue;  // warp-uniform: no row of this warp draws
#pragma unroll 1
    for (int ch = 0; ch < kBN / 32; ++ch) {
      tmem_ld32(tp + ch * 32, v);
      tmem_ld32(tq + ch * 32, w);
      if (draw) {
#pragma unroll
        for (int i = 0; i < 32; ++i)
          mass += fmaxf(ex2_approx(fmaf(v[i], c, -ri.Cp)) - ex2_approx(fmaf(w[i], c, -ri.Cq)), 0.f);
      }
    }
    if (draw) L.mass[(int64_t)row * L.ncta + cta] = mass;
  }
  ok = grid_barrier(L.barrier, 3u * ((unsigned)L.ncta + L.shortfall), a.status, flag,
                    L.max_polls) && ok;

  // ---- epilogue 4: locate the tile holding u_res * Z (warp per row; lane l
  // owns tiles [l*per, (l+1)*per) and keeps their masses in registers; the
  // same arithmetic in every CTA)
  const int32_t per = (L.ncta + 31) / 32;  // <= kMaxTilesPerLane
  for (int m = 0; m < mt && ok; ++m) {
    for (int rl = warp; rl < kBM; rl += kCombWarps) {
      LmSmemRow& ri = rowinfo[m * kBM + rl];
      if (ri.state != 1) continue;
      const int32_t row = m * kBM + rl;
      for (int fp = 0; fp < 2; ++fp) {
        float mk[kMaxTilesPerLane];
#pragma unroll
        for (int q = 0; q < kMaxTilesPerLane; ++q) {
          const int k = lane * per + q;
          mk[q] = 0.f;
          if (q < per && k < L.ncta) {
            if (fp == 0) {
              mk[q] = L.mass[(int64_t)row * L.ncta + k];
            } else {  // masses of p itself, from the tile partials
              const float4 p0 = reinterpret_cast<const float4*>(L.part + (int64_t)row * L.ncta + k)[0];
              mk[q] = p0.y * ex2_approx(p0.x * c - ri.Cp);
            }
          }
        }
        float ls = 0.f;
#pragma unroll
        for (int q = 0; q < kMaxTilesPerLane; ++q) ls += mk[q];
        float incl = ls;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const float y = __shfl_up_sync(0xffffffffu, incl, o);
          if (lane >= o) incl += y;
        }
        const float Z = __shfl_sync(0xffffffffu, incl, 31);
        if (!(Z > 0.f)) {
          if (fp == 1 && lane == 0 && cta == 0) {
            a.out_tok[row] = -1;
            record_status(a.status, SSD_ERR_DEVICE_BOUNDS);
          }
          continue;  // zero residual mass: try p
        }
        const float target = ri.u_res * Z;
        const uint32_t pos = __ballot_sync(0xffffffffu, ls > 0.f);
        const uint32_t cross = __ballot_sync(0xffffffffu, ls > 0.f && incl > target);
        const int32_t lstar = cross ? (__ffs(cross) - 1) : (31 - __clz(pos));
        float t1 = __shfl_sync(0xffffffffu, incl - ls, lstar);
        t1 = cross ? target - t1 : INFINITY;
        if (lane == lstar) {
          int32_t ks = -1, klast = -1;
          float tk = INFINITY, cum = 0.f;
#pragma unroll
          for (int q = 0; q < kMaxTilesPerLane; ++q) {
            if (q < per && lane * per + q < L.ncta) {
              if (mk[q] > 0.f) {
                klast = lane * per + q;
                if (ks < 0 && cum + mk[q] > t1) { ks = klast; tk = t1 - cum; }
              }
              cum += mk[q];
            }
          }
          if (ks < 0) { ks = klast; tk = INFINITY; }
          ri.cstar = ks;
          ri.tc = tk;
          ri.from_p = fp;
        }
        __syncwarp();
        break;
      }
    }
  }
  __syncthreads();

  // ---- epilogue 5: the CTA holding the crossing scans its tile sequentially
  for (int m = 0; m < mt && ok && warp < kTmemWarps; ++m) {
    const int32_t row = m * kBM + tid;
    const LmSmemRow& ri = rowinfo[m * kBM + tid];
    const bool mine = row < rows && ri.state == 1 && ri.cstar == cta;
    if (!__any_sync(0xffffffffu, mine)) continue;  // warp-uniform
    const bool from_p = ri.from_p != 0;
    const uint32_t tp = tmem + lane_off + m * 2 * kBN, tq = tp + kBN;
    float v[32], w[32];
    float cum = 0.f;
    int32_t pick = -1, lastpos = -1;
#pragma unroll 1
    for (int ch = 0; ch < kBN / 32; ++ch) {
      tmem_ld32(tp + ch * 32, v);
      tmem_ld32(tq + ch * 32, w);
      if (mine && pick < 0) {
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const float pv = ex2_approx(fmaf(v[i], c, -ri.Cp));
          const float wt = from_p ? pv : fmaxf(pv - ex2_approx(fmaf(w[i], c, -ri.Cq)), 0.f);
          cum += wt;
          if (wt > 0.f) {
            lastpos = v0 + ch * 32 + i;
            if (pick < 0 && cum > ri.tc) pick = lastpos;
          }
        }
      }
    }
    if (mine) a.out_tok[row] = pick >= 0 ? pick : lastpos;
  }

  // ---- teardown: release TMEM (all MMAs have completed: `done` fired)
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, ncols);
  }
}

// bf16 [outer][inner] matrix, box [box_outer x 64 inner], 128-byte swizzle.
bool make_map(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer,
              uint32_t box_outer) {
  EncodeTiledFn fn = tensor_map_encoder();
  if (fn == nullptr) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {inner * 2};
  cuuint32_t box[2] = {64, box_outer};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// bf16 [K][V] weights as the 3D view {64 vocabulary entries, K rows, V / 64
// column blocks} (the last dimension steps 128 B along a row); a box
// {64, kBK, 2} is one CTA's [2 blocks][kBK rows][128 B] weight tile in one copy.
bool make_weight_map(CUtensorMap* map, const void* base, uint64_t V, uint64_t K) {
  EncodeTiledFn fn = tensor_map_encoder();
  if (fn == nullptr) return false;
  cuuint64_t dims[3] = {64, K, V / 64};
  cuuint64_t strides[2] = {V * 2, 128};
  cuuint32_t box[3] = {64, kBK, kBN / 64};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

size_t al256(size_t x) { return (x + 255) & ~size_t(255); }

int row_tiles(int32_t rows) { return (rows + kBM - 1) / kBM; }

size_t smem_bytes(int mt, int stages) {
  // + the first rejected draft of each sequence (at most one per row)
  return 1024 + (size_t)stages * (2 * mt * kTileA + 2 * kTileB) + (2 * stages + 1) * 8 + 16 +
         (size_t)mt * kBM * sizeof(LmSmemRow) + (size_t)mt * kBM * sizeof(int32_t);
}

// As many stages as the shared memory holds, at most 8.
int stages_for(int mt) {
  int s = 8;
  while (s > 2 && smem_bytes(mt, s) > 232448) --s;
  return s;
}

}  // namespace

size_t lmhead_workspace(int32_t rows, int32_t V) {
  const size_t ncta = (size_t)(V + kBN - 1) / kBN;
  return al256(2 * sizeof(unsigned int)) + al256((size_t)rows * ncta * sizeof(LmPartial)) +
         al256((size_t)rows * ncta * sizeof(float)) + al256((size_t)rows * sizeof(LmRowRec));
}

ssd_status lmhead_check(int32_t rows, int32_t V, int32_t K) {
  if (rows < 1 || rows > kMaxRowTiles * kBM) return SSD_ERR_UNSUPPORTED;
  if (K <= 0 || K % kBK != 0) return SSD_ERR_UNSUPPORTED;
  if (V <= 0 || V % kBN != 0) return SSD_ERR_UNSUPPORTED;
  if (V / kBN > 32 * kMaxTilesPerLane) return SSD_ERR_UNSUPPORTED;
  // every CTA must be resident at once (one CTA per SM: TMEM and shared memory)
  const int mt = row_tiles(rows);
  int per_sm = 0;
  const size_t smem = smem_bytes(mt, stages_for(mt));
  if (cudaFuncSetAttribute(lmhead_accept_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem) != cudaSuccess)
    return SSD_ERR_CUDA;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, lmhead_accept_kernel, kThreadsL,
                                                    smem) != cudaSuccess)
    return SSD_ERR_CUDA;
  if ((int64_t)(V / kBN) > (int64_t)per_sm * device_sm_count()) return SSD_ERR_UNSUPPORTED;
  return SSD_OK;
}

cudaError_t launch_lmhead(const LmHeadArgs& a, void* ws, size_t ws_bytes, cudaStream_t stream) {
  if (a.rows == 0) return cudaSuccess;
  const int mt = row_tiles(a.rows);
  LmLaunch L;
  L.ncta = a.V / kBN;
  L.mt = mt;
  L.stages = stages_for(mt);
  L.max_polls = wait_poll_limit();
  L.shortfall = barrier_shortfall();
  unsigned char* w = static_cast<unsigned char*>(ws);
  L.barrier = reinterpret_cast<unsigned int*>(w);  // [0] arrivals, [1] abort flag
  w += al256(2 * sizeof(unsigned int));
  L.part = reinterpret_cast<LmPartial*>(w);
  w += al256((size_t)a.rows * L.ncta * sizeof(LmPartial));
  L.mass = reinterpret_cast<float*>(w);
  w += al256((size_t)a.rows * L.ncta * sizeof(float));
  L.rec = reinterpret_cast<LmRowRec*>(w);
  CUtensorMap ht, hd, wt, wd;
  // hidden [rows][K]: boxes of 128 rows (rows past `rows` read as zero);
  // weights [K][V]: boxes of 64 K-rows x 128 vocabulary entries (3D view)
  if (!make_map(&ht, a.h_tgt, (uint64_t)a.K, (uint64_t)a.rows, kBM) ||
      !make_map(&hd, a.h_drf, (uint64_t)a.K, (uint64_t)a.rows, kBM) ||
      !make_weight_map(&wt, a.w_tgt, (uint64_t)a.V, (uint64_t)a.K) ||
      !make_weight_map(&wd, a.w_drf, (uint64_t)a.V, (uint64_t)a.K))
    return cudaErrorInvalidValue;
  cudaError_t e = cudaSuccess;
  if (!a.counters_zeroed) {
    e = cudaMemsetAsync(L.barrier, 0, kLmheadCounters * sizeof(unsigned int), stream);
    if (e != cudaSuccess) return e;
  }
  const size_t smem = smem_bytes(mt, L.stages);
  e = cudaFuncSetAttribute(lmhead_accept_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)L.ncta, 1, 1);
  cfg.blockDim = dim3(kThreadsL, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, lmhead_accept_kernel, ht, hd, wt, wd, a, L);
}

}  // namespace ssd
