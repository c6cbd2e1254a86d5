// attention_tc.cu — frontier attention (step a2) on the 5th-generation tensor
// cores.  Same contract as the mma.sync kernel in attention.cu (Sec. 3.3
// "Verification as Auto Correction": the drafted block passes through the
// backbone in parallel; every draft attends to the committed cache and to the
// drafts before it in raster order):
//   O[b][j][h] = softmax_s(scale * Q[b][j][h] . K[b][g][s] + M(s, j)) V[b][g][s]
//
// Design (GB300, tcgen05 + TMEM), one CTA per (KV split, sequence, KV head,
// tile of 128 query rows = drafts x the Hq/Hkv heads sharing the KV head):
//  * warp 8 (producer): Q once through a 3D tensor map, then K and V tiles of
//    64 keys through a 4-stage mbarrier ring (TMA, 128-byte swizzle);
//  * warp 9 (MMA): S_t = Q K_t^T into one of two TMEM S buffers, then, once
//    the softmax has written P_t, O += P_t V_t into the TMEM O accumulator;
//    tcgen05.commit releases each K/V stage and signals each product;
//  * warps 0-7 (softmax; query row = TMEM lane, warp w owns lane quarter w % 4
//    and the half w / 4 of every row's columns): tcgen05.ld of its half of the
//    row of S_t, the spatial mask predicate in registers, the partial maxima of
//    the two halves exchanged through a named barrier per warp pair, the
//    running max and sum, P_t as swizzled bf16 in shared memory (the A operand
//    of the PV product).  Warps whose rows are all padding skip the math.
//    The running max is only moved (and O in TMEM rescaled with tcgen05.ld/st)
//    when it grows by more than 2^8; otherwise the exponentials use the stale
//    max, which the final sum shares, so the result is exact.
// Every barrier a thread waits on is at most one phase ahead of it (S, P and
// PV barriers are per buffer), so parity waits are unambiguous.
#include "kernels.cuh"

namespace ssd {

namespace {

constexpr int kBM = 128;          // query rows per CTA (TMEM lanes)
constexpr int KTC = 64;           // keys per tile
constexpr int kNS = 4;            // K/V ring stages
constexpr int kSoftWarps = 8;     // two per TMEM lane quarter, each taking half of every row
constexpr int kThreadsTC = (kSoftWarps + 2) * 32;
constexpr float kLog2eTC = 1.4426950408889634f;
constexpr float kRescale = 8.0f;  // log2 growth of the running max that forces a rescale

__device__ __forceinline__ void tmem_alloc_tc(uint32_t* dst, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(dst)),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish_tc() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_tc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tc_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void umma(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                     uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   smem_u32(bar))
               : "memory");
}
__device__ __forceinline__ void tld32(uint32_t taddr, float* v) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,"
      "%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void tst32(uint32_t taddr, const float* v) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
      "%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
      "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
      "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
      "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
      "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
      "r"(__float_as_uint(v[15])), "r"(__float_as_uint(v[16])), "r"(__float_as_uint(v[17])),
      "r"(__float_as_uint(v[18])), "r"(__float_as_uint(v[19])), "r"(__float_as_uint(v[20])),
      "r"(__float_as_uint(v[21])), "r"(__float_as_uint(v[22])), "r"(__float_as_uint(v[23])),
      "r"(__float_as_uint(v[24])), "r"(__float_as_uint(v[25])), "r"(__float_as_uint(v[26])),
      "r"(__float_as_uint(v[27])), "r"(__float_as_uint(v[28])), "r"(__float_as_uint(v[29])),
      "r"(__float_as_uint(v[30])), "r"(__float_as_uint(v[31]))
      : "memory");
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ float ex2a(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// tcgen05 shared-memory descriptor: 128-byte swizzle, version 1.
__device__ __forceinline__ uint64_t sdesc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

// kind::f16 instruction descriptor: fp32 D, bf16 A and B, A K-major, M = 128.
__host__ __device__ constexpr uint32_t idesc_f16(int n, bool b_mn_major) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (0u << 15) | ((b_mn_major ? 1u : 0u) << 16) |
         ((uint32_t)(n >> 3) << 17) | ((uint32_t)(kBM >> 4) << 24);
}

struct TcLaunch {
  int32_t splits, kps, mtiles;
  float* part_o;
  float* part_lse;
  int32_t* seq_ok;
};

template <int D>
constexpr size_t tc_smem_bytes() {
  return 1024 + (size_t)kBM * D * 2 + (size_t)2 * kNS * KTC * D * 2 + (size_t)2 * kBM * KTC * 2 +
         256 + 132 * 4 + (size_t)4 * kBM * 4 + 16;
}

template <int D>
__global__ void __launch_bounds__(kThreadsTC, 1)
frontier_attn_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                        const __grid_constant__ CUtensorMap tmV, AttnArgs a, TcLaunch L) {
  constexpr int NSUB = D / 64;
  constexpr int Q_BYTES = kBM * D * 2;
  constexpr int KV_BYTES = KTC * D * 2;      // one K (or V) tile
  constexpr int P_BYTES = kBM * KTC * 2;     // one P buffer
  constexpr uint32_t kIdescS = idesc_f16(KTC, false);
  constexpr uint32_t kIdescO = idesc_f16(D, true);
  constexpr uint32_t kTmemCols = 256;        // S x 2 (64 each) + O (<= 128)
  constexpr int HC = KTC / 2;                // S columns per softmax thread
  constexpr int HD = D / 2;                  // O columns per softmax thread

  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  unsigned char* sQ = smem;
  unsigned char* sK = sQ + Q_BYTES;                 // [kNS][KV_BYTES]
  unsigned char* sV = sK + kNS * KV_BYTES;          // [kNS][KV_BYTES]
  unsigned char* sP = sV + kNS * KV_BYTES;          // [2][P_BYTES]
  uint64_t* bar = reinterpret_cast<uint64_t*>(sP + 2 * P_BYTES);
  uint64_t* q_full = bar;
  uint64_t* kv_full = bar + 1;                      // [kNS]
  uint64_t* kv_empty = kv_full + kNS;               // [kNS]
  uint64_t* s_full = kv_empty + kNS;                // [2]
  uint64_t* s_free = s_full + 2;                    // [2]
  uint64_t* p_full = s_free + 2;                    // [2]
  uint64_t* pv_done = p_full + 2;                   // [2]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(pv_done + 2);
  int32_t* kflat = reinterpret_cast<int32_t*>(tmem_slot + 4);  // [128]
  int32_t* bad = kflat + 128;
  float* xch = reinterpret_cast<float*>(bad + 4);   // [2 parities][2 halves][128 rows]

  __shared__ int32_t s_order[kLptMax + 1];
  const int32_t split = blockIdx.x;
  const int32_t bg = blockIdx.y;
  const int32_t g = bg % a.Hkv;
  const int32_t b = longest_first(a, bg / a.Hkv, s_order);
  const int32_t G = a.Hq / a.Hkv;
  const int32_t tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

  const int32_t cache = a.cache_len[b];
  const int32_t nd = a.n_drafts[b];
  const int32_t Lk = cache + nd;
  const bool shape_ok = !(nd < 0 || nd > a.D_max || cache < 0 || Lk > a.L_max);
  const int32_t rows_total = shape_ok ? nd * G : 0;
  const int32_t row0 = blockIdx.z * kBM;
  const int32_t k_lo = split * L.kps;
  const int32_t k_hi = min(Lk, k_lo + L.kps);
  const bool has_work = shape_ok && nd > 0 && row0 < rows_total && k_lo < Lk;
  const int32_t ntiles = has_work ? (k_hi - k_lo + KTC - 1) / KTC : 0;
  const int32_t n_active = (Lk + L.kps - 1) / L.kps;

  // ---- draft positions (validity is identical in every CTA of b)
  if (tid == 0) *bad = shape_ok ? 0 : 1;
  __syncthreads();
  bool seq_valid = shape_ok;
  if (shape_ok) {
    const int32_t HW = a.grid.grid_h * a.grid.grid_w;
    for (int32_t j = tid; j < nd; j += blockDim.x) {
      const int32_t gidx = a.draft_pos[(int64_t)b * a.D_max + j];
      if (gidx < 0 || gidx >= HW) {
        *bad = 1;
        kflat[j] = 0;
      } else {
        const int32_t y = gidx / a.grid.grid_w, x = gidx - y * a.grid.grid_w;
        kflat[j] = a.grid.prefix_len + y * a.grid.row_stride + x;
      }
    }
    __syncthreads();
    seq_valid = (*bad == 0);
  }
  if (split == 0 && g == 0 && blockIdx.z == 0 && tid == 0) {
    L.seq_ok[b] = seq_valid ? 1 : 0;
    if (!seq_valid) record_status(a.status, SSD_ERR_DEVICE_BOUNDS);
  }
  if (!seq_valid || !has_work) return;

  // ---- set-up: barriers, TMEM
  if (tid == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < kNS; ++s) {
      mbar_init(&kv_full[s], 1);
      mbar_init(&kv_empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s_full[i], 1);
      mbar_init(&s_free[i], kSoftWarps);
      mbar_init(&p_full[i], kSoftWarps);
      mbar_init(&pv_done[i], 1);
    }
    fence_barrier_init();
  }
  if (warp == 0) {
    tmem_alloc_tc(tmem_slot, kTmemCols);
    tmem_relinquish_tc();
  }
  tc_before();
  __syncthreads();
  tc_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t tS = tmem, tO = tmem + 2 * KTC;

  const float c2 = (a.scale != 0.f ? a.scale : rsqrtf((float)D)) * kLog2eTC;
  const int32_t kvrow0 = (b * a.Hkv + g) * a.L_max + k_lo;  // 2D row of the first key

  if (warp == kSoftWarps) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      const uint64_t polq = policy_evict_last();
      mbar_arrive_expect_tx(q_full, Q_BYTES);
      for (int c = 0; c < NSUB; ++c) {
        // 3D Q view {d, Hq, B * D_max}: box {64, G, 128 / G} -> rows (j, hg)
        asm volatile(
            "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
            " [%0], [%1, {%2, %3, %4}], [%5], %6;" ::"r"(smem_u32(sQ + c * (kBM * 128))),
            "l"(reinterpret_cast<uint64_t>(&tmQ)), "r"(c * 64), "r"(g * G),
            "r"(b * a.D_max + row0 / G), "r"(smem_u32(q_full)), "l"(polq)
            : "memory");
      }
      for (int t = 0; t < ntiles; ++t) {
        const int s = t % kNS;
        if (t >= kNS && !mbar_wait(&kv_empty[s], ((t / kNS) - 1) & 1, a.status)) break;
        mbar_arrive_expect_tx(&kv_full[s], 2 * KV_BYTES);
        const int32_t row = kvrow0 + t * KTC;
        for (int c = 0; c < NSUB; ++c) {
          tma_load_2d(sK + s * KV_BYTES + c * (KTC * 128), &tmK, c * 64, row, &kv_full[s], pol);
          tma_load_2d(sV + s * KV_BYTES + c * (KTC * 128), &tmV, c * 64, row, &kv_full[s], pol);
        }
      }
    }
    __syncwarp();
  } else if (warp == kSoftWarps + 1) {
    // ----------------------------------------------------------------- MMA
    if (lane == 0) {
      bool ok = mbar_wait(q_full, 0, a.status);
      const uint32_t q0 = smem_u32(sQ);
      auto issue_pv = [&](int t) {
        const int bb = t & 1, s = t % kNS;
        if (!mbar_wait(&p_full[bb], (t >> 1) & 1, a.status)) return false;
        tc_after();
        const uint32_t p0 = smem_u32(sP + bb * P_BYTES);
        const uint32_t v0 = smem_u32(sV + s * KV_BYTES);
#pragma unroll
        for (int kk = 0; kk < KTC / 16; ++kk) {
          // A = P (K-major, 128-byte rows), B = V (MN-major: d atoms KTC*128 bytes
          // apart, 8-key groups 1 KB apart; 16 keys = 2 KB per step)
          umma(tO, sdesc(p0 + kk * 32, 16, 1024), sdesc(v0 + kk * 2048, KTC * 128, 1024), kIdescO,
               (t > 0 || kk > 0) ? 1u : 0u);
        }
        umma_commit(&kv_empty[s]);
        umma_commit(&pv_done[bb]);
        return true;
      };
      for (int t = 0; t < ntiles && ok; ++t) {
        const int s = t % kNS, bb = t & 1;
        if (!mbar_wait(&kv_full[s], (t / kNS) & 1, a.status)) { ok = false; break; }
        if (t >= 2 && !mbar_wait(&s_free[bb], ((t >> 1) - 1) & 1, a.status)) { ok = false; break; }
        tc_after();
        const uint32_t k0 = smem_u32(sK + s * KV_BYTES);
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
          const int sub = ks >> 2, kin = (ks & 3) * 32;
          umma(tS + bb * KTC, sdesc(q0 + sub * (kBM * 128) + kin, 16, 1024),
               sdesc(k0 + sub * (KTC * 128) + kin, 16, 1024), kIdescS, ks > 0 ? 1u : 0u);
        }
        umma_commit(&s_full[bb]);
        if (t >= 1 && !issue_pv(t - 1)) { ok = false; break; }
      }
      if (ok && ntiles > 0) issue_pv(ntiles - 1);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------- softmax
    const int quarter = warp & 3, half = warp >> 2;
    const int32_t rl = quarter * 32 + lane;   // row inside the tile = TMEM lane
    const int32_t r = row0 + rl;              // this thread's query row
    const bool live = r < rows_total;
    const bool warp_live = row0 + quarter * 32 < rows_total;  // same for both warps of a pair
    const int32_t qpos = live ? kflat[r / G] : 0x7fffffff;
    // cache slots below every query position of this CTA are visible to all rows
    int32_t minq = 0x7fffffff;
    for (int32_t rr = row0; rr < min(rows_total, row0 + kBM); ++rr) minq = min(minq, kflat[rr / G]);
    const int32_t mask_from = min(cache, minq + 1);
    const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
    float m_run = -INFINITY, l_run = 0.f;  // l_run: this half's partial sum
    bool ok = true;
    // partial values of the two halves of a row, double-buffered by tile parity
    auto xslot = [&](int parity, int hf) -> float& { return xch[(parity * 2 + hf) * kBM + rl]; };
    auto pair_sync = [&]() { asm volatile("bar.sync %0, 64;" ::"r"(1 + quarter) : "memory"); };
    for (int t = 0; t < ntiles; ++t) {
      const int bb = t & 1;
      if (!mbar_wait(&s_full[bb], (t >> 1) & 1, a.status)) ok = false;
      tc_after();
      float sv[HC];
      if (warp_live) tld32(tS + lane_off + bb * KTC + half * HC, sv);
      tc_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&s_free[bb]);
      bool moved = false;
      float alpha = 1.f;
      uint32_t pk[HC / 2];
      if (warp_live) {
        // mask: keys past this split / the sequence, and the spatial predicate
        const int32_t c0 = k_lo + t * KTC + half * HC;
        if (c0 + HC > k_hi || c0 + HC > mask_from) {
#pragma unroll
          for (int jj = 0; jj < HC; ++jj) {
            const int32_t key = c0 + jj;
            const int32_t kp = key < cache ? key : (key < Lk ? kflat[key - cache] : 0x7fffffff);
            if (!(key < k_hi && kp <= qpos)) sv[jj] = -INFINITY;
          }
        }
        float mx = -INFINITY;
#pragma unroll
        for (int jj = 0; jj < HC; ++jj) mx = fmaxf(mx, sv[jj]);
        xslot(bb, half) = mx;
        pair_sync();
        mx = fmaxf(mx, xslot(bb, half ^ 1));
        // move the running max only when it grows by more than 2^kRescale
        if (mx != -INFINITY && (m_run == -INFINITY || (mx - m_run) * c2 > kRescale)) {
          alpha = (m_run == -INFINITY) ? 0.f : ex2a((m_run - mx) * c2);
          m_run = mx;
          moved = true;
        }
        const float moff = (m_run == -INFINITY) ? 0.f : m_run * c2;
        float rs = 0.f;
#pragma unroll
        for (int jj = 0; jj < HC; jj += 2) {
          const float e0 = ex2a(fmaf(sv[jj], c2, -moff));
          const float e1 = ex2a(fmaf(sv[jj + 1], c2, -moff));
          rs += e0 + e1;
          pk[jj / 2] = pack_bf16x2(e0, e1);
        }
        l_run = l_run * alpha + rs;
      }
      // P_t may overwrite the buffer PV(t-2) read; O may be rescaled once PV(t-1) is done
      if (t >= 2 && !mbar_wait(&pv_done[bb], ((t >> 1) - 1) & 1, a.status)) ok = false;
      if (warp_live) {
        unsigned char* prow = sP + bb * P_BYTES + rl * 128;
#pragma unroll
        for (int cq = 0; cq < HC / 8; ++cq) {  // 16-byte chunks of this half
          const int cch = half * (HC / 8) + cq;
          const uint4 v4 = make_uint4(pk[4 * cq], pk[4 * cq + 1], pk[4 * cq + 2], pk[4 * cq + 3]);
          *reinterpret_cast<uint4*>(prow + ((cch ^ (rl & 7)) << 4)) = v4;
        }
        if (__any_sync(0xffffffffu, moved && t > 0)) {
          if (!mbar_wait(&pv_done[(t - 1) & 1], ((t - 1) >> 1) & 1, a.status)) ok = false;
          tc_after();
          float ov[32];
#pragma unroll 1
          for (int cc = 0; cc < HD / 32; ++cc) {
            const uint32_t ta = tO + lane_off + half * HD + cc * 32;
            tld32(ta, ov);
#pragma unroll
            for (int i = 0; i < 32; ++i) ov[i] *= alpha;
            tst32(ta, ov);
          }
        }
      }
      fence_proxy_async();  // P stores -> visible to the tensor core
      tc_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_full[bb]);
    }
    // ---- epilogue: wait for the last PV product, normalise, write this half
    if (ntiles > 0 && !mbar_wait(&pv_done[(ntiles - 1) & 1], ((ntiles - 1) >> 1) & 1, a.status))
      ok = false;
    tc_after();
    if (warp_live) {
      xslot(ntiles & 1, half) = l_run;  // the parity the last tile did not use
      pair_sync();
      const float l_tot = l_run + xslot(ntiles & 1, half ^ 1);
      const float inv_l = l_tot > 0.f ? 1.0f / l_tot : 0.f;
      const float lse = (l_tot > 0.f) ? (m_run * (c2 / kLog2eTC) + logf(l_tot)) : -INFINITY;
      const bool direct = (n_active == 1);
      const int32_t jq = live ? r / G : 0, h = g * G + (live ? r % G : 0);
#pragma unroll 1
      for (int cc = 0; cc < HD / 32; ++cc) {
        float ov[32];
        tld32(tO + lane_off + half * HD + cc * 32, ov);
        if (!live || !ok) continue;
        const int col = half * HD + cc * 32;
        if (direct) {
          __nv_bfloat16* ob = reinterpret_cast<__nv_bfloat16*>(a.o) +
                              (((int64_t)b * a.D_max + jq) * a.Hq + h) * D + col;
#pragma unroll
          for (int i = 0; i < 32; i += 8) {
            uint4 w;
            w.x = pack_bf16x2(ov[i] * inv_l, ov[i + 1] * inv_l);
            w.y = pack_bf16x2(ov[i + 2] * inv_l, ov[i + 3] * inv_l);
            w.z = pack_bf16x2(ov[i + 4] * inv_l, ov[i + 5] * inv_l);
            w.w = pack_bf16x2(ov[i + 6] * inv_l, ov[i + 7] * inv_l);
            *reinterpret_cast<uint4*>(ob + i) = w;
          }
        } else {
          const int64_t prow = (((int64_t)b * a.Hq + h) * a.D_max + jq) * L.splits + split;
          float* po = L.part_o + prow * D + col;
#pragma unroll
          for (int i = 0; i < 32; i += 4)
            *reinterpret_cast<float4*>(po + i) =
                make_float4(ov[i] * inv_l, ov[i + 1] * inv_l, ov[i + 2] * inv_l, ov[i + 3] * inv_l);
        }
      }
      if (live && ok && half == 0) {
        if (direct) {
          if (a.lse != nullptr) a.lse[((int64_t)b * a.Hq + h) * a.D_max + jq] = lse;
        } else {
          L.part_lse[(((int64_t)b * a.Hq + h) * a.D_max + jq) * L.splits + split] = lse;
        }
      }
    }
  }
  // ---- teardown
  tc_before();
  __syncthreads();
  if (warp == 0) {
    tc_after();
    tmem_dealloc_tc(tmem, kTmemCols);
  }
}

typedef CUresult (*EncodeTiledFnTc)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                    const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                    const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                    CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFnTc encode_tc() {
  static EncodeTiledFnTc fn = nullptr;
  if (fn == nullptr) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFnTc>(p);
  }
  return fn;
}

}  // namespace

bool attention_tc_supported(int32_t Hq, int32_t Hkv, int32_t d, int32_t D_max) {
  const int32_t G = Hq / Hkv;
  // Below 64 query rows per KV group the 128-row MMA tile is mostly padding and
  // the mma.sync kernel (several CTAs per SM) is faster.
  return (d == 64 || d == 128) && G >= 1 && G <= kBM && (kBM % G) == 0 && D_max * G > 64;
}

TcPlan attention_tc_plan(int32_t B, int32_t Hq, int32_t Hkv, int32_t D_max, int32_t L_max) {
  TcPlan p;
  const int32_t G = Hq / Hkv;
  p.mtiles = (D_max * G + kBM - 1) / kBM;
  const int64_t base = (int64_t)B * Hkv * p.mtiles;
  const int32_t target = device_sm_count();  // one CTA per SM
  const int32_t max_splits = max(1, (L_max + 2 * KTC - 1) / (2 * KTC));  // >= 2 tiles each
  int32_t splits = (int32_t)((target + base - 1) / base);
  splits = max(1, min(splits, max_splits));
  int32_t kps = (L_max + splits - 1) / splits;
  kps = ((kps + KTC - 1) / KTC) * KTC;
  p.splits = (L_max + kps - 1) / kps;
  p.kps = kps;
  return p;
}

cudaError_t launch_attention_tc(const AttnArgs& a, const TcPlan& p, int32_t* seq_ok, float* part_o,
                                float* part_lse, cudaStream_t stream) {
  EncodeTiledFnTc fn = encode_tc();
  if (fn == nullptr) return cudaErrorInvalidValue;
  const int32_t G = a.Hq / a.Hkv;
  CUtensorMap tq, tk, tv;
  {
    cuuint64_t dims[3] = {(cuuint64_t)a.d, (cuuint64_t)a.Hq, (cuuint64_t)a.B * a.D_max};
    cuuint64_t strides[2] = {(cuuint64_t)a.d * 2, (cuuint64_t)a.Hq * a.d * 2};
    cuuint32_t box[3] = {64, (cuuint32_t)G, (cuuint32_t)(kBM / G)};
    cuuint32_t estr[3] = {1, 1, 1};
    if (fn(&tq, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(a.q), dims, strides, box,
           estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  const int64_t rows = (int64_t)a.B * a.Hkv * a.L_max;
  for (int w = 0; w < 2; ++w) {
    cuuint64_t dims[2] = {(cuuint64_t)a.d, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)a.d * 2};
    cuuint32_t box[2] = {64, KTC};
    cuuint32_t estr[2] = {1, 1};
    if (fn(w == 0 ? &tk : &tv, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
           const_cast<void*>(w == 0 ? a.k : a.v), dims, strides, box, estr,
           CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  TcLaunch L;
  L.splits = p.splits;
  L.kps = p.kps;
  L.mtiles = p.mtiles;
  L.part_o = part_o;
  L.part_lse = part_lse;
  L.seq_ok = seq_ok;
  const dim3 grid(p.splits, a.B * a.Hkv, p.mtiles);
  const dim3 block(kThreadsTC);
  cudaError_t e;
  if (a.d == 128) {
    const size_t smem = tc_smem_bytes<128>();
    e = cudaFuncSetAttribute(frontier_attn_tc_kernel<128>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    frontier_attn_tc_kernel<128><<<grid, block, smem, stream>>>(tq, tk, tv, a, L);
  } else {
    const size_t smem = tc_smem_bytes<64>();
    e = cudaFuncSetAttribute(frontier_attn_tc_kernel<64>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    frontier_attn_tc_kernel<64><<<grid, block, smem, stream>>>(tq, tk, tv, a, L);
  }
  return cudaGetLastError();
}

}  // namespace ssd
