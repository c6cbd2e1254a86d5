// attention.cu — frontier attention (step a2): every draft query of a
// sequence attends to the committed KV cache plus the drafted block's own
// keys under the spatial dependency mask (Sec. 3.3 "Verification as Auto
// Correction": the drafted block passes through the backbone in parallel;
// App. "Deviation from AR": a draft's context may hold other drafts).
//
//   O[b][j][h] = softmax_s(scale * Q[b][j][h] . K[b][g][s] + M(s, j)) V[b][g][s]
//   M(s, j) = 0 iff pos(s) <= pos(j), pos(s) = s for cache slots s < cache_len,
//   pos(cache_len + j') = prefix + y' * row_stride + x' of draft j'.
//
// Design (GB300): one CTA per (KV split, sequence b, KV head g, query tile),
// sequences taken longest first.  All draft queries of the KV group (drafts x
// the Hq/Hkv query heads sharing g) sit in the CTA's warps, 16 query rows per
// warp, so each K/V tile is read from HBM once per KV head.  K/V tiles of 64
// keys are staged by TMA (2D tensor maps, 128-byte swizzle, evict-first L2
// policy) through a 2-stage mbarrier ring (three CTAs per SM); QK^T and PV
// run as mma.sync (bf16 inputs, fp32 accumulation), the mask predicate is
// evaluated in registers only on tiles that reach the drafted block, and the
// softmax is the online (running max / running sum) form with quad shuffles.
// Long caches are split over CTAs; a combine kernel merges the splits by
// their log-sum-exp.

#include "kernels.cuh"

namespace ssd {

namespace {

#ifndef SSD_ATTN_CTAS_PER_SM
#define SSD_ATTN_CTAS_PER_SM 2  // KV splits are added until the grid has this many CTAs per SM
#endif
#ifndef SSD_ATTN_STAGES
#define SSD_ATTN_STAGES 2  // K/V ring depth: 2 lets three CTAs share an SM
#endif
constexpr int KT = 64;        // keys per tile
constexpr int kStages = SSD_ATTN_STAGES;
constexpr int kMaxWarps = 8;  // 128 query rows per CTA
constexpr float kLog2e = 1.4426950408889634f;

// ------------------------------------------------------------ PTX wrappers
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void mma_bf16(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Byte offset of 16-byte chunk `ch` of row `row` inside a [rows x 128 B]
// TMA box written with CU_TENSOR_MAP_SWIZZLE_128B (1024-byte aligned base).
__device__ __forceinline__ uint32_t swz(int row, int ch) {
  return (uint32_t)(row * 128 + ((ch ^ (row & 7)) << 4));
}

struct AttnLaunch {
  int32_t splits;        // KV splits (host-chosen)
  int32_t kps;           // keys per split, multiple of KT
  int32_t nwarps;        // warps per CTA (16 query rows each)
  float* part_o;         // [B][Hq][D_max][splits][d] fp32 (splits > 1)
  float* part_lse;       // [B][Hq][D_max][splits]
  int32_t* seq_ok;       // [B] 1 if the sequence's inputs were in range
};

// Validity of one sequence's frontier; identical in every CTA of b.
__device__ __forceinline__ bool load_draft_positions(const AttnArgs& a, int32_t b, int32_t nd,
                                                     int32_t* kflat, int32_t* bad) {
  const int32_t HW = a.grid.grid_h * a.grid.grid_w;
  for (int32_t j = threadIdx.x; j < nd; j += blockDim.x) {
    const int32_t gidx = attn_draft_pos(a, b, j);
    if (gidx < 0 || gidx >= HW) {
      *bad = 1;
      kflat[j] = 0;
    } else {
      const int32_t y = gidx / a.grid.grid_w, x = gidx - y * a.grid.grid_w;
      kflat[j] = a.grid.prefix_len + y * a.grid.row_stride + x;
    }
  }
  __syncthreads();
  return *bad == 0;
}

// Launched as a programmatic dependent (the step's schedule): block 0 exits
// only after the kernel before it, and lets the next kernel be scheduled
// then, so that stream order holds.
__device__ __forceinline__ void pdl_exit() {
  if (pdl_first_block()) {
    pdl_wait();
    pdl_launch_dependents();
  }
}

template <int D>
__global__ void __launch_bounds__(kMaxWarps * 32, 1)
frontier_attn_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                     AttnArgs a, AttnLaunch L) {
  constexpr int NSUB = D / 64;                 // 128-byte column boxes per row
  constexpr int TILE_BYTES = KT * D * 2;       // one K (or V) tile
  constexpr int KSTEPS = D / 16;               // k16 steps of QK^T
  constexpr int NT_O = D / 8;                  // n8 tiles of O
  // as in the tcgen05 kernel: a dependent may start beside it once block 0
  // has seen the kernel before this one complete (block 0 triggers on exit)
  if (!pdl_first_block()) pdl_launch_dependents();
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  // 1024-byte alignment for the swizzle atoms
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  unsigned char* sK = smem;                                  // [stages][TILE]
  unsigned char* sV = smem + kStages * TILE_BYTES;           // [stages][TILE]
  uint64_t* full = reinterpret_cast<uint64_t*>(sV + kStages * TILE_BYTES);
  int32_t* kflat = reinterpret_cast<int32_t*>(full + kStages);  // [128]
  int32_t* bad = kflat + 128;

  __shared__ int32_t s_order[kLptMax + 1];
  const int32_t split = blockIdx.x;
  const int32_t bg = blockIdx.y;
  const int32_t g = bg % a.Hkv;
  const int32_t b = longest_first(a, bg / a.Hkv, s_order);
  const int32_t G = a.Hq / a.Hkv;
  const int32_t tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

  const int32_t cache = a.cache_len[b];
  const int32_t nd = attn_drafts(a, b);
  const int32_t Lk = cache + nd;
  const bool shape_ok = !(nd < 0 || nd > a.D_max || cache < 0 || Lk > a.L_max);
  const int32_t rows_total = shape_ok ? nd * G : 0;
  const int32_t row0 = blockIdx.z * (L.nwarps * 16);
  const int32_t k_lo = split * L.kps;
  const int32_t k_hi = min(Lk, k_lo + L.kps);
  // CTAs with keys and query rows of a well-formed sequence start streaming
  // K/V right away, before the dependent loads of the draft positions and Q
  const bool has_work = shape_ok && nd > 0 && row0 < rows_total && k_lo < Lk;
  const int32_t ntiles = has_work ? (k_hi - k_lo + KT - 1) / KT : 0;
  const int32_t n_active = (Lk + L.kps - 1) / L.kps;  // splits holding keys of b

  const uint64_t policy = policy_evict_first();
  const int32_t kvrow0 = (b * a.Hkv + g) * a.L_max;  // row of slot 0 in the 2D view
  if (tid == 0 && has_work) {
    for (int s = 0; s < kStages; ++s) mbar_init(&full[s], 1);
    fence_barrier_init();
  }
  __syncthreads();
  auto issue = [&](int t) {
    const int s = t % kStages;
    mbar_arrive_expect_tx(&full[s], 2 * TILE_BYTES);
    const int32_t row = kvrow0 + k_lo + t * KT;
    // one copy per tile: for d = 128 the map is the 3D view {64, rows, 2}
    if constexpr (NSUB == 2) {
      tma_load_3d(sK + s * TILE_BYTES, &tmK, 0, row, 0, &full[s], policy);
      tma_load_3d(sV + s * TILE_BYTES, &tmV, 0, row, 0, &full[s], policy);
    } else {
      tma_load_2d(sK + s * TILE_BYTES, &tmK, 0, row, &full[s], policy);
      tma_load_2d(sV + s * TILE_BYTES, &tmV, 0, row, &full[s], policy);
    }
  };
  const int32_t n_pre = min(kStages - 1, ntiles);
  if (tid == 0) {
    for (int t = 0; t < n_pre; ++t) issue(t);
  }

  // ---- draft positions (validity is identical in every CTA of b)
  if (tid == 0) *bad = shape_ok ? 0 : 1;
  __syncthreads();
  const bool seq_valid = shape_ok && load_draft_positions(a, b, nd, kflat, bad);
  if (split == 0 && g == 0 && blockIdx.z == 0 && tid == 0) {
    L.seq_ok[b] = seq_valid ? 1 : 0;
    if (!seq_valid) record_status(a.status, SSD_ERR_DEVICE_BOUNDS);
  }
  if (!seq_valid || !has_work) {
    // never leave with copies in flight into this CTA's shared memory
    for (int t = 0; t < n_pre; ++t) mbar_wait(&full[t % kStages], 0, a.status);
    pdl_exit();
    return;
  }

  // ---- rows of this warp: r = row0 + warp * 16 + {lane/4, lane/4 + 8}
  const int32_t wrow = row0 + warp * 16;
  const bool warp_active = wrow < rows_total;
  int32_t qpos[2];
  int32_t rr[2];
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    rr[i] = wrow + (lane >> 2) + 8 * i;
    qpos[i] = (rr[i] < rows_total) ? kflat[rr[i] / G] : 0x7fffffff;
  }
  // first key index whose visibility is not implied (cache slots below every
  // query position of this CTA are visible to all of its rows)
  int32_t minq = 0x7fffffff;
  for (int32_t r = row0; r < min(rows_total, row0 + L.nwarps * 16); ++r)
    minq = min(minq, kflat[r / G]);
  const int32_t mask_from = min(cache, minq + 1);

  // ---- Q fragments (A operand of QK^T), straight from global memory
  uint32_t qf[KSTEPS][4];
  {
    const __nv_bfloat16* qb = reinterpret_cast<const __nv_bfloat16*>(a.q);
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const int32_t r = rr[i];
      const bool live = r < rows_total;
      const int32_t j = live ? r / G : 0, h = g * G + (live ? r % G : 0);
      const uint32_t* src =
          reinterpret_cast<const uint32_t*>(qb + (((int64_t)b * a.D_max + j) * a.Hq + h) * D);
#pragma unroll
      for (int ks = 0; ks < KSTEPS; ++ks) {
        const int col = ks * 16 + (lane & 3) * 2;
        qf[ks][i] = live ? src[col / 2] : 0u;
        qf[ks][2 + i] = live ? src[(col + 8) / 2] : 0u;
      }
    }
  }

  const float c2 = (a.scale != 0.f ? a.scale : rsqrtf((float)D)) * kLog2e;
  float o[NT_O][4];
#pragma unroll
  for (int n = 0; n < NT_O; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;
  float m_run[2] = {-INFINITY, -INFINITY};
  float l_run[2] = {0.f, 0.f};
  bool ok = true;

  for (int t = 0; t < ntiles; ++t) {
    if (tid == 0 && t + kStages - 1 < ntiles) issue(t + kStages - 1);
    const int s = t % kStages;
    if (!mbar_wait(&full[s], (t / kStages) & 1, a.status)) ok = false;
    if (warp_active && ok) {
      const uint32_t kbase = smem_u32(sK + s * TILE_BYTES);
      const uint32_t vbase = smem_u32(sV + s * TILE_BYTES);
      // ---- S = Q K^T for 16 rows x 64 keys
      float sc[8][4];
#pragma unroll
      for (int n = 0; n < 8; ++n) sc[n][0] = sc[n][1] = sc[n][2] = sc[n][3] = 0.f;
#pragma unroll
      for (int ks = 0; ks < KSTEPS; ++ks) {
        const int sub = ks >> 2, cb = (ks & 3) * 2;
#pragma unroll
        for (int np = 0; np < 4; ++np) {  // pairs of n8 tiles: keys np*16 .. +15
          const int mi = lane >> 3;
          const int key = np * 16 + (lane & 7) + ((mi >> 1) << 3);
          const int ch = cb + (mi & 1);
          uint32_t b0, b1, b2, b3;
          ldsm_x4(kbase + sub * (KT * 128) + swz(key, ch), b0, b1, b2, b3);
          mma_bf16(sc[2 * np], qf[ks][0], qf[ks][1], qf[ks][2], qf[ks][3], b0, b1);
          mma_bf16(sc[2 * np + 1], qf[ks][0], qf[ks][1], qf[ks][2], qf[ks][3], b2, b3);
        }
      }
      // ---- mask: keys past this split / the sequence, and the spatial predicate
      const int32_t tile0 = k_lo + t * KT;
      if (tile0 + KT > k_hi || tile0 + KT > mask_from) {
#pragma unroll
        for (int n = 0; n < 8; ++n) {
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const int32_t key = tile0 + n * 8 + (lane & 3) * 2 + (e & 1);
            const int32_t kp = key < cache ? key : (key < Lk ? kflat[key - cache] : 0x7fffffff);
            const bool vis = key < k_hi && kp <= qpos[e >> 1];
            if (!vis) sc[n][e] = -INFINITY;
          }
        }
      }
      // ---- online softmax (rows lane/4 and lane/4 + 8; quads share a row)
      float alpha[2];
#pragma unroll
      for (int i = 0; i < 2; ++i) {
        float mx = -INFINITY;
#pragma unroll
        for (int n = 0; n < 8; ++n) mx = fmaxf(mx, fmaxf(sc[n][2 * i], sc[n][2 * i + 1]));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
        const float m_new = fmaxf(m_run[i], mx);
        const float m_use = (m_new == -INFINITY) ? 0.f : m_new;
        alpha[i] = exp2f((m_run[i] - m_use) * c2);  // 0 when nothing was accumulated
        m_run[i] = m_new;
        const float moff = m_use * c2;
        float rs = 0.f;
#pragma unroll
        for (int n = 0; n < 8; ++n) {
          sc[n][2 * i] = exp2f(fmaf(sc[n][2 * i], c2, -moff));
          sc[n][2 * i + 1] = exp2f(fmaf(sc[n][2 * i + 1], c2, -moff));
          rs += sc[n][2 * i] + sc[n][2 * i + 1];
        }
        rs += __shfl_xor_sync(0xffffffffu, rs, 1);
        rs += __shfl_xor_sync(0xffffffffu, rs, 2);
        l_run[i] = l_run[i] * alpha[i] + rs;
      }
#pragma unroll
      for (int n = 0; n < NT_O; ++n) {
        o[n][0] *= alpha[0];
        o[n][1] *= alpha[0];
        o[n][2] *= alpha[1];
        o[n][3] *= alpha[1];
      }
      // ---- O += P V (P re-packed from the S accumulators as A fragments)
#pragma unroll
      for (int kk = 0; kk < KT / 16; ++kk) {
        const uint32_t a0 = pack_bf16x2(sc[2 * kk][0], sc[2 * kk][1]);
        const uint32_t a1 = pack_bf16x2(sc[2 * kk][2], sc[2 * kk][3]);
        const uint32_t a2 = pack_bf16x2(sc[2 * kk + 1][0], sc[2 * kk + 1][1]);
        const uint32_t a3 = pack_bf16x2(sc[2 * kk + 1][2], sc[2 * kk + 1][3]);
#pragma unroll
        for (int np = 0; np < NT_O / 2; ++np) {  // pairs of n8 tiles: d cols np*16 .. +15
          const int mi = lane >> 3;
          const int key = kk * 16 + (lane & 7) + ((mi & 1) << 3);
          const int dc = np * 16 + ((mi >> 1) << 3);  // first d column of the 8x8 block
          const int sub = dc >> 6, ch = (dc & 63) >> 3;
          uint32_t b0, b1, b2, b3;
          ldsm_x4_t(vbase + sub * (KT * 128) + swz(key, ch), b0, b1, b2, b3);
          mma_bf16(o[2 * np], a0, a1, a2, a3, b0, b1);
          mma_bf16(o[2 * np + 1], a0, a1, a2, a3, b2, b3);
        }
      }
    }
    // stage s is free for the producer; a timed-out wait anywhere stops every thread
    if (!__syncthreads_and(ok)) { ok = false; break; }
  }
  if (!ok || !warp_active) {
    pdl_exit();
    return;
  }

  // ---- epilogue: normalise, write O (bf16) or the split partial (fp32)
  const bool direct = (n_active == 1);
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int32_t r = rr[i];
    if (r >= rows_total) continue;
    const int32_t j = r / G, h = g * G + r % G;
    const float inv_l = l_run[i] > 0.f ? 1.0f / l_run[i] : 0.f;
    const float lse = (l_run[i] > 0.f) ? (m_run[i] * (c2 / kLog2e) + logf(l_run[i])) : -INFINITY;
    // (debug builds: the row's store index against its buffer)
    if (direct ? !dbg_in(((int64_t)b * a.D_max + j) * a.Hq + h, (int64_t)a.B * a.D_max * a.Hq,
                         a.status)
               : !dbg_in((((int64_t)b * a.Hq + h) * a.D_max + j) * L.splits + split,
                         (int64_t)a.B * a.Hq * a.D_max * L.splits, a.status))
      continue;
    if (direct) {
      __nv_bfloat16* ob = reinterpret_cast<__nv_bfloat16*>(a.o) +
                          (((int64_t)b * a.D_max + j) * a.Hq + h) * D;
#pragma unroll
      for (int n = 0; n < NT_O; ++n) {
        const int col = n * 8 + (lane & 3) * 2;
        *reinterpret_cast<uint32_t*>(ob + col) =
            pack_bf16x2(o[n][2 * i] * inv_l, o[n][2 * i + 1] * inv_l);
      }
      if (a.lse != nullptr && (lane & 3) == 0)
        a.lse[((int64_t)b * a.Hq + h) * a.D_max + j] = lse;
    } else {
      const int64_t prow = (((int64_t)b * a.Hq + h) * a.D_max + j) * L.splits + split;
      float* po = L.part_o + prow * D;
#pragma unroll
      for (int n = 0; n < NT_O; ++n) {
        const int col = n * 8 + (lane & 3) * 2;
        *reinterpret_cast<float2*>(po + col) = make_float2(o[n][2 * i] * inv_l, o[n][2 * i + 1] * inv_l);
      }
      if ((lane & 3) == 0) L.part_lse[prow] = lse;
    }
  }
  pdl_exit();
}

// One warp per (b, j, h) row: merge the active splits by log-sum-exp.
template <int D>
__global__ void attn_combine_kernel(AttnArgs a, AttnLaunch L) {
  const int64_t gw = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int32_t lane = threadIdx.x & 31;
  const int64_t total = (int64_t)a.B * a.D_max * a.Hq;
  if (gw >= total) return;
  const int32_t h = (int32_t)(gw % a.Hq);
  const int32_t j = (int32_t)((gw / a.Hq) % a.D_max);
  const int32_t b = (int32_t)(gw / ((int64_t)a.Hq * a.D_max));
  if (!L.seq_ok[b]) return;
  const int32_t nd = attn_drafts(a, b);
  if (j >= nd) return;
  const int32_t Lk = a.cache_len[b] + nd;
  const int32_t n_active = (Lk + L.kps - 1) / L.kps;
  if (n_active <= 1) return;  // written directly by the attention kernel
  const int64_t prow = (((int64_t)b * a.Hq + h) * a.D_max + j) * L.splits;
  if (!dbg_in(prow + n_active - 1, (int64_t)a.B * a.Hq * a.D_max * L.splits, a.status)) return;
  float mx = -INFINITY;
  for (int s = 0; s < n_active; ++s) mx = fmaxf(mx, L.part_lse[prow + s]);
  constexpr int PER = D / 32;
  float acc[PER];
#pragma unroll
  for (int k = 0; k < PER; ++k) acc[k] = 0.f;
  float wsum = 0.f;
  for (int s = 0; s < n_active; ++s) {
    const float ls = L.part_lse[prow + s];
    const float w = (ls == -INFINITY) ? 0.f : expf(ls - mx);
    wsum += w;
    const float* po = L.part_o + (prow + s) * D + lane * PER;
#pragma unroll
    for (int k = 0; k < PER; ++k) acc[k] += w * po[k];
  }
  const float inv = 1.0f / wsum;
  __nv_bfloat16* ob =
      reinterpret_cast<__nv_bfloat16*>(a.o) + (((int64_t)b * a.D_max + j) * a.Hq + h) * D + lane * PER;
#pragma unroll
  for (int k = 0; k < PER; k += 2)
    *reinterpret_cast<uint32_t*>(ob + k) = pack_bf16x2(acc[k] * inv, acc[k + 1] * inv);
  if (a.lse != nullptr && lane == 0) a.lse[((int64_t)b * a.Hq + h) * a.D_max + j] = mx + logf(wsum);
}

// ------------------------------------------------------------- host side
// View of a bf16 [B][Hkv][L_max][d] tensor whose box is one K (or V) tile of
// KT rows in the layout [d / 64][KT rows][128 B]: for d = 128 the 3D view
// {64 columns, rows, 2 halves} with the halves 128 B apart inside a row; for
// d = 64 the 2D view {64, rows}.
bool make_kv_map(CUtensorMap* map, const void* base, int64_t rows, int32_t d) {
  EncodeTiledFn fn = tensor_map_encoder();
  if (fn == nullptr) return false;
  const cuuint32_t rank = d == 128 ? 3 : 2;
  cuuint64_t dims[3] = {64, (cuuint64_t)rows, 2};
  cuuint64_t strides[2] = {(cuuint64_t)d * 2, 128};
  cuuint32_t box[3] = {64, KT, 2};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void*>(base), dims, strides,
            box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

struct Plan {
  int32_t nwarps, mtiles, splits, kps;
  bool tc;  // tcgen05 kernel (attention_tc.cu)
};

// `rows_hint` (<= D_max) bounds the drafts a sequence can have in this launch;
// it chooses between the two kernels only, both of which size their work by
// D_max, so a wrong hint costs time, never correctness.
Plan make_plan(int32_t B, int32_t Hq, int32_t Hkv, int32_t d, int32_t D_max, int32_t L_max,
               int32_t rows_hint) {
  Plan p;
  p.tc = attention_tc_supported(Hq, Hkv, d, min(D_max, rows_hint));
  if (p.tc) {
    const TcPlan t = attention_tc_plan(B, Hq, Hkv, D_max, L_max);
    p.nwarps = 0;
    p.mtiles = t.mtiles;
    p.splits = t.splits;
    p.kps = t.kps;
    return p;
  }
  const int32_t G = Hq / Hkv;
  const int32_t rows = D_max * G;
  p.nwarps = min(kMaxWarps, (rows + 15) / 16);
  p.mtiles = (rows + p.nwarps * 16 - 1) / (p.nwarps * 16);
  const int64_t base = (int64_t)B * Hkv * p.mtiles;
  const int32_t target = SSD_ATTN_CTAS_PER_SM * device_sm_count();
  const int32_t max_splits = max(1, (L_max + 2 * KT - 1) / (2 * KT));  // >= 2 tiles per split
  int32_t splits = (int32_t)((target + base - 1) / base);
  splits = max(1, min(splits, max_splits));
  int32_t kps = (L_max + splits - 1) / splits;
  kps = ((kps + KT - 1) / KT) * KT;
  p.splits = (L_max + kps - 1) / kps;
  p.kps = kps;
  return p;
}

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

}  // namespace

EncodeTiledFn tensor_map_encoder() {
  static EncodeTiledFn fn = nullptr;
  if (fn == nullptr) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

bool bf16_tensor_map(CUtensorMap* map, const void* base, uint32_t rank, const uint64_t* dims,
                     const uint64_t* strides, const uint32_t* box) {
  EncodeTiledFn fn = tensor_map_encoder();
  if (fn == nullptr || rank < 1 || rank > 5) return false;
  cuuint64_t d[5], s[4];
  cuuint32_t b[5], e[5];
  for (uint32_t i = 0; i < rank; ++i) {
    d[i] = dims[i];
    b[i] = box[i];
    e[i] = 1;
    if (i + 1 < rank) s[i] = strides[i];
  }
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void*>(base), d, s, b, e,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int device_sm_count() {
  int dev = 0, n = 0;
  cudaGetDevice(&dev);
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
  return n;
}

int32_t attention_rows_hint(const ssd_grid& g, int32_t D_max) {
  if (g.grid_w <= 0 || g.k_h < 0 || g.k_v < 0) return D_max;
  const int64_t h = g.k_h > 0 ? min(g.k_h, g.grid_w) : g.grid_w;
  const int64_t n = h + (int64_t)g.k_v * g.grid_w;
  return n < D_max ? (int32_t)n : D_max;
}

// Large enough for the plan of either kernel, so that the kernel choice (which
// depends on the grid) never outgrows a workspace sized without it.
size_t attention_workspace(int32_t B, int32_t Hq, int32_t Hkv, int32_t d, int32_t D_max,
                           int32_t L_max) {
  size_t bytes = align256((size_t)B * sizeof(int32_t));
  int32_t splits = 1;
  for (int32_t hint : {D_max, 0}) splits = max(splits, make_plan(B, Hq, Hkv, d, D_max, L_max, hint).splits);
  if (splits > 1) {
    const size_t prow = (size_t)B * Hq * D_max * splits;
    bytes += align256(prow * d * sizeof(float)) + align256(prow * sizeof(float));
  }
  return bytes;
}

static cudaError_t launch_combine(const AttnArgs& a, const AttnLaunch& L, cudaStream_t stream);

int attention_launches(const ssd_grid& g, int32_t B, int32_t Hq, int32_t Hkv, int32_t d,
                       int32_t D_max, int32_t L_max) {
  if (B == 0) return 0;
  return make_plan(B, Hq, Hkv, d, D_max, L_max, attention_rows_hint(g, D_max)).splits > 1 ? 2 : 1;
}

namespace {

// The launch record of a plan over workspace `ws` (laid out as attention_workspace counts it).
AttnLaunch carve(const AttnArgs& a, const Plan& p, void* ws) {
  AttnLaunch L;
  L.splits = p.splits;
  L.kps = p.kps;
  L.nwarps = p.nwarps;
  unsigned char* w = static_cast<unsigned char*>(ws);
  L.seq_ok = reinterpret_cast<int32_t*>(w);
  w += align256((size_t)a.B * sizeof(int32_t));
  L.part_o = nullptr;
  L.part_lse = nullptr;
  if (p.splits > 1) {
    const size_t prow = (size_t)a.B * a.Hq * a.D_max * p.splits;
    L.part_o = reinterpret_cast<float*>(w);
    w += align256(prow * a.d * sizeof(float));
    L.part_lse = reinterpret_cast<float*>(w);
  }
  return L;
}

}  // namespace

cudaError_t launch_attention_combine(const AttnArgs& a, void* ws, cudaStream_t stream) {
  if (a.B == 0) return cudaSuccess;
  const Plan p = make_plan(a.B, a.Hq, a.Hkv, a.d, a.D_max, a.L_max,
                           attention_rows_hint(a.grid, a.D_max));
  return p.splits == 1 ? cudaSuccess : launch_combine(a, carve(a, p, ws), stream);
}

cudaError_t launch_attention(const AttnArgs& a, void* ws, size_t ws_bytes, cudaStream_t stream,
                             bool defer_combine, bool pdl) {
  if (a.B == 0) return cudaSuccess;
  const Plan p = make_plan(a.B, a.Hq, a.Hkv, a.d, a.D_max, a.L_max,
                           attention_rows_hint(a.grid, a.D_max));
  const AttnLaunch L = carve(a, p, ws);
  cudaError_t e;
  if (p.tc) {
    e = launch_attention_tc(a, TcPlan{p.splits, p.kps, p.mtiles}, L.seq_ok, L.part_o, L.part_lse,
                            stream, pdl);
    if (e != cudaSuccess) return e;
    return (p.splits == 1 || defer_combine) ? cudaSuccess : launch_combine(a, L, stream);
  }
  CUtensorMap tmK, tmV;
  const int64_t rows = (int64_t)a.B * a.Hkv * a.L_max;
  if (!make_kv_map(&tmK, a.k, rows, a.d) || !make_kv_map(&tmV, a.v, rows, a.d))
    return cudaErrorInvalidValue;
  const dim3 grid(p.splits, a.B * a.Hkv, p.mtiles);
  const dim3 block(p.nwarps * 32);
  if (a.d == 128) {
    const size_t smem = 1024 + kStages * 2 * (KT * 128 * 2) + kStages * 8 + 129 * 4;
    e = cudaFuncSetAttribute(frontier_attn_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
    if (e != cudaSuccess) return e;
    e = launch_kernel(frontier_attn_kernel<128>, grid, block, smem, stream, false, tmK, tmV, a, L);
    if (e != cudaSuccess) return e;
  } else {
    const size_t smem = 1024 + kStages * 2 * (KT * 64 * 2) + kStages * 8 + 129 * 4;
    e = cudaFuncSetAttribute(frontier_attn_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
    if (e != cudaSuccess) return e;
    e = launch_kernel(frontier_attn_kernel<64>, grid, block, smem, stream, false, tmK, tmV, a, L);
    if (e != cudaSuccess) return e;
  }
  e = cudaGetLastError();
  if (e != cudaSuccess || p.splits == 1 || defer_combine) return e;
  return launch_combine(a, L, stream);
}

static cudaError_t launch_combine(const AttnArgs& a, const AttnLaunch& L, cudaStream_t stream) {
  const int64_t rows_c = (int64_t)a.B * a.D_max * a.Hq;
  const int wpb = 8;
  const unsigned blocks = (unsigned)((rows_c + wpb - 1) / wpb);
  if (a.d == 128)
    attn_combine_kernel<128><<<blocks, wpb * 32, 0, stream>>>(a, L);
  else
    attn_combine_kernel<64><<<blocks, wpb * 32, 0, stream>>>(a, L);
  return cudaGetLastError();
}

// ------------------------------------------------- no-allocation variant
// Scratch of ssd_verify_attention_noalloc(): it stands in for the caller's
// workspace (per-sequence flags and split-KV partials).  Host code must not
// pass `g_noalloc_scratch` itself to a kernel: on the host that name is a
// stand-in, not a device address.  Every call looks the device address up
// below, with the caller's device current.
static __device__ __align__(256) unsigned char g_noalloc_scratch[SSD_NOALLOC_SCRATCH_BYTES];

namespace {

// Device address of the scratch array on the current device, or nullptr.  The
// first look-up on a device is its set-up (it may load the library's device
// code there); later ones are a host-side table look-up.  Looking it up on
// every call, rather than caching it, means a device reset (which reloads the
// module, possibly elsewhere) can never leave a stale address behind.
void* noalloc_scratch() {
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess) return nullptr;
  return p;
}

}  // namespace

cudaError_t launch_attention_noalloc(const AttnArgs& a, cudaStream_t stream) {
  const size_t need = attention_workspace(a.B, a.Hq, a.Hkv, a.d, a.D_max, a.L_max);
  if (need > SSD_NOALLOC_SCRATCH_BYTES) return cudaErrorMemoryAllocation;
  void* ws = noalloc_scratch();
  if (ws == nullptr) return cudaErrorInvalidDevice;
  return launch_attention(a, ws, SSD_NOALLOC_SCRATCH_BYTES, stream);
}

}  // namespace ssd
