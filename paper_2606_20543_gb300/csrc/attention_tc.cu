// attention_tc.cu — frontier attention (step a2) on the 5th-generation tensor
// cores.  Same contract as the mma.sync kernel in attention.cu (Sec. 3.3
// "Verification as Auto Correction": the drafted block passes through the
// backbone in parallel; every draft attends to the committed cache and to the
// drafts before it in raster order):
//   O[b][j][h] = softmax_s(scale * Q[b][j][h] . K[b][g][s] + M(s, j)) V[b][g][s]
//
// Design (GB300, tcgen05 + TMEM): a persistent kernel, one CTA per SM, that
// walks work items (KV split, sequence, KV head, tile of 128 query rows =
// drafts x the Hq/Hkv heads sharing the KV head; 64-row tiles with M = 64
// products when a KV head's query rows fit in 64).  Sequences are taken
// longest first and the items are dealt to the CTAs in snake order, so the
// long items start early and every CTA gets a similar share.
//  * warp 8 (producer): decodes the next item, checks and converts its draft
//    positions into an item slot (two slots), loads Q into one of two Q
//    buffers through a 3D tensor map, then the item's K tiles of 128 keys;
//    warp 10 streams its V tiles (TMA, 128-byte swizzle, one copy per tile,
//    issued by two threads because one thread issues only a few million copies
//    per second).  The producers run ahead of the other warps by up to two
//    items, so the next item's loads overlap the current item's last tiles
//    and its epilogue;
//  * warp 9 issues S_t = Q K_t^T (N = 128 keys) into one of two TMEM S/P
//    buffers; warp 11, once the softmax has written P_t, O += P_t V_t with P
//    read from TMEM (the A operand of a tcgen05.mma may live in tensor
//    memory) into the item's TMEM O buffer (two buffers, so an item's
//    epilogue overlaps the next item's products);
//  * warps 0-7 (softmax; query row = TMEM lane, warp w owns lane quarter w % 4
//    and the half w / 4 of every row's columns): tcgen05.ld of its half of the
//    row of S_t, the spatial mask (a per-row bitmask of the visible drafts,
//    built once per item), the partial maxima of the two halves exchanged
//    through a named barrier per warp pair, the running max and sum, and P_t
//    as bf16 pairs stored with tcgen05.st over the first half of the same
//    TMEM buffer; then the item's epilogue.  Warps whose rows are all padding
//    skip the math.  The running max is only moved (and O in TMEM rescaled
//    with tcgen05.ld/st) when it grows by more than 2^8; otherwise the
//    exponentials use the stale max, which the final sum shares, so the
//    result is exact.
// K stages, V stages and S/P buffers form rings of two indexed by tile t mod
// 2, and one barrier per ring slot covers several conditions: "K_t loaded and
// S/P buffer free (PV of tile t - 2 done)" and "V_t loaded and P_t written".
// An mbarrier poll costs a few hundred cycles even when the phase is complete
// and a tcgen05.mma tens of cycles to issue, so each issuing thread has one
// wait, one group of products and one commit per 128-key tile.  Code that
// runs once per item (mask, bitmask, epilogue) is kept small: unrolled cold
// paths cost instruction-cache misses of thousands of cycles.
// Every barrier a thread waits on is at most one phase ahead of it (tile
// barriers are per tile parity, item barriers per item slot), so parity
// waits are unambiguous.
#include <algorithm>

#include "kernels.cuh"

namespace ssd {

namespace {

constexpr int kBM = 128;          // query rows per CTA (TMEM lanes)
constexpr int KTC = 128;          // keys per tile
constexpr int kNB = 2;            // ring depth: K stages, V stages, TMEM S/P buffers
constexpr uint32_t kTmemCols = 512;  // S/P x 2 (128 columns each), O x 2 (128 columns each) at 256
constexpr int kSoftWarps = 8;     // two per TMEM lane quarter, each taking half of every row
constexpr int kThreadsTC = (kSoftWarps + 4) * 32;  // + K/Q producer, S, V producer, PV
constexpr float kLog2eTC = 1.4426950408889634f;
constexpr float kRescale = 8.0f;  // log2 growth of the running max that forces a rescale

// 16-lane TMEM accesses of the M = 64 products, whose row m sits in lane
// 32 (m / 16) + m % 16.  .16x256b: thread t holds rows t/4 and t/4 + 8 of the
// 16 lanes, columns 8u + 2 (t % 4) + {0, 1} of unit u, as registers 4u + {0, 1}
// (row t/4) and 4u + {2, 3} (row t/4 + 8).  .16x128b: column 4u + t % 4 of
// unit u, register 2u (row t/4) and 2u + 1 (row t/4 + 8).
__device__ __forceinline__ void tld16x256_x8(uint32_t taddr, float* v) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.16x256b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
      "%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
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
__device__ __forceinline__ void tld16x256_x4(uint32_t taddr, float* v) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.16x256b.x4.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
      "%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr)
      : "memory");
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void tst16x256_x8(uint32_t taddr, const float* v) {
  asm volatile(
      "tcgen05.st.sync.aligned.16x256b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
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
__device__ __forceinline__ void tst16x256_x4(uint32_t taddr, const float* v) {
  asm volatile(
      "tcgen05.st.sync.aligned.16x256b.x4.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
      "%14,%15,%16};" ::"r"(taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
      "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
      "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
      "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
      "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
      "r"(__float_as_uint(v[15]))
      : "memory");
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tst16x128_x8(uint32_t taddr, const uint32_t* v) {
  asm volatile(
      "tcgen05.st.sync.aligned.16x128b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
      "%14,%15,%16};" ::"r"(taddr),
      "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]),
      "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15])
      : "memory");
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// kind::f16 instruction descriptor: fp32 D, bf16 A and B, A K-major, M = m (64 or 128).
__host__ __device__ constexpr uint32_t idesc_f16(int n, bool b_mn_major, int m = kBM) {
  return idesc_bf16(m, n, false, b_mn_major);
}

struct TcLaunch {
  int32_t splits, kps, mtiles;
  float* part_o;
  float* part_lse;
  int32_t* seq_ok;
};

// One work item (KV split, sequence, KV head, query tile) as the producer
// hands it to the MMA and softmax warps; ntiles < 0 ends the CTA's work.
struct TcItem {
  int32_t b, g, split, row0, rows_total, cache, Lk, k_lo, k_hi, ntiles, direct;
  int32_t increasing;  // kflat strictly increasing (the raster frontier): draft j sees draft j' iff j' <= j
  int32_t pad[4];
  int32_t kflat[128];  // raster position of each draft of b
};

template <int D, int BM>
constexpr size_t tc_smem_bytes() {
  return 1024 + (size_t)2 * BM * D * 2 + (size_t)2 * kNB * KTC * D * 2 + 320 +
         2 * sizeof(TcItem) + (size_t)6 * kBM * 4;
}

// One K or V tile of KTC keys in the MMA's layout [d / 64][KTC rows][128 B]
// (128-byte swizzle) with one copy: for d = 128 the tensor map is the 3D view
// {64, rows, 2} whose last dimension steps 128 B inside a row.
template <int D>
__device__ __forceinline__ void load_kv_tile(void* dst, const CUtensorMap* map, int32_t row,
                                             uint64_t* bar, uint64_t pol) {
  if constexpr (D == 128)
    tma_load_3d(dst, map, 0, row, 0, bar, pol);
  else
    tma_load_2d(dst, map, 0, row, bar, pol);
}

// BM = 128: query tiles of 128 rows, row m in TMEM lane m.  BM = 64 (items of
// at most 64 query rows): M = 64 products, row m in lane 32 (m / 16) + m % 16,
// so the rows spread over the four lane quarters and their softmax over all
// four SM sub-partitions.
template <int D, int BM>
__global__ void __launch_bounds__(kThreadsTC, 1)
frontier_attn_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                        const __grid_constant__ CUtensorMap tmV, AttnArgs a, TcLaunch L) {
  static_assert(BM == 64 || BM == 128, "query tile");
  constexpr int NSUB = D / 64;
  constexpr int Q_BYTES = BM * D * 2;
  constexpr int KV_BYTES = KTC * D * 2;      // one K (or V) tile
  constexpr uint32_t kIdescS = idesc_f16(KTC, false, BM);
  constexpr uint32_t kIdescO = idesc_f16(D, true, BM);
  constexpr int HC = KTC / 2;                // S columns per softmax thread (P: HC / 2)
  constexpr int HD = D / 2;                  // O columns per softmax thread

  extern __shared__ __align__(1024) unsigned char smem_raw[];
  __shared__ int32_t s_order[kLptMax];
  __shared__ int32_t s_key[kLptMax];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  unsigned char* sQ = smem;                         // [2][Q_BYTES]
  unsigned char* sK = sQ + 2 * Q_BYTES;             // [kNB][KV_BYTES]
  unsigned char* sV = sK + kNB * KV_BYTES;          // [kNB][KV_BYTES]
  uint64_t* bar = reinterpret_cast<uint64_t*>(sV + kNB * KV_BYTES);
  uint64_t* q_full = bar;                           // [2] per item slot
  uint64_t* q_empty = q_full + 2;                   // [2]
  uint64_t* it_full = q_empty + 2;                  // [2]
  uint64_t* it_empty = it_full + 2;                 // [2]
  uint64_t* o_empty = it_empty + 2;                 // [2]
  // per ring slot t % kNB: k_ready = K_t loaded and the TMEM S/P buffer free
  // (PV_{t-kNB} done); s_full = S_t done (K stage free); v_ready = V_t loaded
  // and P_t written; pv_done = PV_t done (V stage free)
  uint64_t* k_ready = o_empty + 2;                  // [kNB]
  uint64_t* s_full = k_ready + kNB;                 // [kNB]
  uint64_t* v_ready = s_full + kNB;                 // [kNB]
  uint64_t* pv_done = v_ready + kNB;                // [kNB]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(pv_done + kNB);
  TcItem* items = reinterpret_cast<TcItem*>(bar + 40);  // [2]
  float* xch = reinterpret_cast<float*>(items + 2);     // [3 slots][2 halves][128 rows]

  const int32_t G = a.Hq / a.Hkv;
  const int32_t tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int32_t per_b = a.Hkv * L.splits * L.mtiles;
  const int64_t n_items = (int64_t)a.B * per_b;

  // ---- set-up: barriers, TMEM, the longest-first order of the sequences
  if (tid == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(&q_full[i], 1);
      mbar_init(&q_empty[i], 1);
      mbar_init(&it_full[i], 1);
      mbar_init(&it_empty[i], kSoftWarps);
      mbar_init(&o_empty[i], kSoftWarps);
    }
    for (int s = 0; s < kNB; ++s) {
      mbar_init(&k_ready[s], 2);
      mbar_init(&s_full[s], 1);
      mbar_init(&v_ready[s], 1 + kSoftWarps);
      mbar_init(&pv_done[s], 1);
    }
    fence_barrier_init();
    // every S/P buffer starts free: the PV arrivals of the first round
    for (int s = 0; s < kNB; ++s) mbar_arrive(&k_ready[s]);
  }
  if (warp == kSoftWarps && lane < 3)  // the first copies need the descriptors
    prefetch_tensormap(lane == 0 ? &tmQ : (lane == 1 ? &tmK : &tmV));
  if (warp == 0) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  if (a.B <= kLptMax) {
    // s_order[rank] = the sequence with the rank-th most keys (ties by index);
    // a sequence with no drafts ranks last (its items are empty)
    for (int32_t i = tid; i < a.B; i += blockDim.x) {
      const int32_t c = a.cache_len[i], n = attn_drafts(a, i);
      s_key[i] = (c >= 0 && n > 0 && c <= a.L_max && n <= a.D_max) ? c + n : 0;
    }
    __syncthreads();
    for (int32_t i = tid; i < a.B; i += blockDim.x) {
      const int32_t key = s_key[i];
      int32_t r = 0;
      for (int32_t j = 0; j < a.B; ++j) {
        const int32_t kj = s_key[j];
        r += (kj > key) || (kj == key && j < i);
      }
      s_order[r] = i;
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t tS = tmem;            // [kNB] x KTC columns: S_t in fp32, then P_t in bf16
  const uint32_t tO0 = tmem + 256;     // [2] x 128 columns

  const float c2 = (a.scale != 0.f ? a.scale : rsqrtf((float)D)) * kLog2eTC;

  if (warp == kSoftWarps) {
    // ------------------------------------------------------------ producer
    // Items in snake order over the longest-first list: round k takes items
    // k * gridDim.x + (blockIdx.x, or its mirror on odd rounds).
    const uint64_t pol = policy_evict_first();
    const uint64_t polq = policy_evict_last();
    const int32_t HW = a.grid.grid_h * a.grid.grid_w;
    bool ok = true;
    int32_t k = 0;        // items handed out
    uint32_t T = 0;       // K/V tiles issued
    for (int64_t round = 0; ok; ++round) {
      const int64_t base = round * gridDim.x;
      if (base >= n_items) break;
      const int64_t i = base + ((round & 1) ? (gridDim.x - 1 - blockIdx.x) : blockIdx.x);
      if (i >= n_items) continue;
      const int32_t rank_b = (int32_t)(i / per_b);
      int32_t rem = (int32_t)(i - (int64_t)rank_b * per_b);
      const int32_t mtile = rem % L.mtiles;
      rem /= L.mtiles;
      const int32_t split = rem % L.splits, g = rem / L.splits;
      const int32_t b = (a.B <= kLptMax) ? s_order[rank_b] : rank_b;
      const int32_t cache = a.cache_len[b], nd = attn_drafts(a, b);
      const bool shape_ok = nd >= 0 && nd <= a.D_max && cache >= 0 && cache <= a.L_max - nd;
      // draft positions (validity is identical in every item of b)
      int32_t kfv[4];
      bool bad = !shape_ok;
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int32_t j = lane + 32 * u;
        kfv[u] = 0;
        if (shape_ok && j < nd) {
          const int32_t gidx = attn_draft_pos(a, b, j);
          if (gidx < 0 || gidx >= HW) {
            bad = true;
          } else {
            const int32_t y = gidx / a.grid.grid_w, x = gidx - y * a.grid.grid_w;
            kfv[u] = a.grid.prefix_len + y * a.grid.row_stride + x;
          }
        }
      }
      const bool valid = !__any_sync(0xffffffffu, bad);
      // strictly increasing positions? (the previous draft of j = lane + 32 u is
      // lane - 1 of the same u, or lane 31 of u - 1)
      bool dec = false;
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int32_t up = __shfl_up_sync(0xffffffffu, kfv[u], 1);
        const int32_t prev_hi = __shfl_sync(0xffffffffu, u > 0 ? kfv[u > 0 ? u - 1 : 0] : 0, 31);
        const int32_t prev = lane > 0 ? up : prev_hi;
        const int32_t j = lane + 32 * u;
        if (j >= 1 && j < nd && kfv[u] <= prev) dec = true;
      }
      const bool increasing = !__any_sync(0xffffffffu, dec);
      if (split == 0 && g == 0 && mtile == 0 && lane == 0) {
        L.seq_ok[b] = valid ? 1 : 0;
        if (!valid) record_status(a.status, SSD_ERR_DEVICE_BOUNDS);
      }
      const int32_t Lk = valid ? cache + nd : 0;
      const int32_t rows_total = valid ? nd * G : 0;
      const int32_t row0 = mtile * BM;
      const int32_t k_lo = split * L.kps;
      const int32_t k_hi = min(Lk, k_lo + L.kps);
      if (!valid || nd == 0 || row0 >= rows_total || k_lo >= Lk) continue;
      const int32_t ntiles = (k_hi - k_lo + KTC - 1) / KTC;
      const int s = k & 1;
      if (k >= 2 && lane == 0) ok = mbar_wait(&it_empty[s], ((k >> 1) - 1) & 1, a.status);
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      TcItem& it = items[s];
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (lane + 32 * u < nd) it.kflat[lane + 32 * u] = kfv[u];
      if (lane == 0) {
        it.b = b;
        it.g = g;
        it.split = split;
        it.row0 = row0;
        it.rows_total = rows_total;
        it.cache = cache;
        it.Lk = Lk;
        it.k_lo = k_lo;
        it.k_hi = k_hi;
        it.ntiles = ntiles;
        it.direct = ((Lk + L.kps - 1) / L.kps) == 1;
        it.increasing = increasing ? 1 : 0;
      }
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&it_full[s]);
        // Q of this item into slot s once the S products of item k - 2 are done
        if (k >= 2) ok = mbar_wait(&q_empty[s], ((k >> 1) - 1) & 1, a.status);
        if (ok) {
          mbar_arrive_expect_tx(&q_full[s], Q_BYTES);
          for (int c = 0; c < NSUB; ++c) {
            // 3D Q view {d, Hq, B * D_max}: box {64, G, BM / G} -> rows (j, hg)
            asm volatile(
                "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
                " [%0], [%1, {%2, %3, %4}], [%5], %6;" ::"r"(
                    smem_u32(sQ + s * Q_BYTES + c * (BM * 128))),
                "l"(reinterpret_cast<uint64_t>(&tmQ)), "r"(c * 64), "r"(g * G),
                "r"(b * a.D_max + row0 / G), "r"(smem_u32(&q_full[s])), "l"(polq)
                : "memory");
          }
        }
        const int32_t kvrow0 = (b * a.Hkv + g) * a.L_max + k_lo;  // 2D row of the first key
        for (int t = 0; t < ntiles && ok; ++t, ++T) {
          const int sb = T % kNB;
          // K stage sb is free once S_{T-kNB} is done
          if (T >= (uint32_t)kNB && !mbar_wait(&s_full[sb], ((T / kNB) - 1) & 1, a.status)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&k_ready[sb], KV_BYTES);
          load_kv_tile<D>(sK + sb * KV_BYTES, &tmK, kvrow0 + t * KTC, &k_ready[sb], pol);
        }
      }
      ok = __shfl_sync(0xffffffffu, ok, 0);
      T = __shfl_sync(0xffffffffu, T, 0);
      ++k;
    }
    if (ok) {
      // end marker
      const int s = k & 1;
      if (k >= 2 && lane == 0) ok = mbar_wait(&it_empty[s], ((k >> 1) - 1) & 1, a.status);
      if (lane == 0 && ok) {
        items[s].ntiles = -1;
        mbar_arrive(&it_full[s]);
      }
    }
    __syncwarp();
  } else if (warp == kSoftWarps + 2) {
    // ---------------------------------------------------------- V producer
    // Follows the item slots like the MMA warp; a slot is not rewritten before
    // the softmax has finished its item, which needs every V tile of it.
    // Launch ordering (programmatic dependent launch): launched as a dependent
    // of the step's acceptance pass, whose results it does not read, the
    // kernel starts as the acceptance's CTAs retire; lane 1 of block 0 waits
    // for the acceptance to complete and only then lets the kernel queued
    // after this one (the counts and draws, which read them) be scheduled
    // beside it; lane 1 of the other blocks lets it be scheduled at once (it
    // is scheduled when every block has).  Under a plain launch the wait
    // returns at once.  The wait sits in the
    // other branch of the V loop's lane test, so that lane 0 never waits at
    // the reconvergence point of a block of its own.
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      uint32_t T = 0;
      bool ok = true;
      for (int32_t k = 0; ok; ++k) {
        const int s = k & 1;
        if (!mbar_wait(&it_full[s], (k >> 1) & 1, a.status)) break;
        const TcItem& it = items[s];
        const int32_t ntiles = it.ntiles;
        if (ntiles < 0) break;
        const int32_t kvrow0 = (it.b * a.Hkv + it.g) * a.L_max + it.k_lo;
        for (int t = 0; t < ntiles; ++t, ++T) {
          const int sb = T % kNB;
          // V stage sb is free once PV_{T-kNB} is done
          if (T >= (uint32_t)kNB && !mbar_wait(&pv_done[sb], ((T / kNB) - 1) & 1, a.status)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&v_ready[sb], KV_BYTES);
          load_kv_tile<D>(sV + sb * KV_BYTES, &tmV, kvrow0 + t * KTC, &v_ready[sb], pol);
        }
      }
    } else if (lane == 1) {
      if (pdl_first_block()) pdl_wait();
      pdl_launch_dependents();
    }
    __syncwarp();
  } else if (warp == kSoftWarps + 1) {
    // ----------------------------------------------------------- S products
    if (lane == 0) {
      uint32_t T = 0;
      for (int32_t k = 0;; ++k) {
        const int s = k & 1;
        if (!mbar_wait(&it_full[s], (k >> 1) & 1, a.status)) break;
        const int32_t ntiles = items[s].ntiles;
        if (ntiles < 0) break;
        if (!mbar_wait(&q_full[s], (k >> 1) & 1, a.status)) break;
        tc_fence_after();
        const uint64_t dq = smem_desc(smem_u32(sQ + s * Q_BYTES), 16, 1024);
        bool ok = true;
        for (int t = 0; t < ntiles; ++t, ++T) {
          const int sb = T % kNB;
          if (!mbar_wait(&k_ready[sb], (T / kNB) & 1, a.status)) { ok = false; break; }
          tc_fence_after();
          const uint64_t dk = smem_desc(smem_u32(sK + sb * KV_BYTES), 16, 1024);
#pragma unroll
          for (int ks = 0; ks < D / 16; ++ks) {
            const int sub = ks >> 2, kin = (ks & 3) * 32;
            mma_ss(tS + sb * KTC, smem_desc_at(dq, sub * (BM * 128) + kin),
                 smem_desc_at(dk, sub * (KTC * 128) + kin), kIdescS, ks > 0 ? 1u : 0u);
          }
          mma_commit(&s_full[sb]);
          if (t == ntiles - 1) mma_commit(&q_empty[s]);
        }
        if (!ok) break;
      }
    }
    __syncwarp();
  } else if (warp == kSoftWarps + 3) {
    // ---------------------------------------------------------- PV products
    // Issued by a thread of its own: a tcgen05.mma takes tens of cycles to
    // issue and an mbarrier poll a few hundred, so one thread issuing both
    // products would be the slowest stage of the tile loop.
    if (lane == 0) {
      uint32_t T = 0;
      for (int32_t k = 0;; ++k) {
        const int s = k & 1;
        if (!mbar_wait(&it_full[s], (k >> 1) & 1, a.status)) break;
        const int32_t ntiles = items[s].ntiles;
        if (ntiles < 0) break;
        // the first product of the item overwrites O[s]: the epilogue of item k - 2 must be done
        if (k >= 2 && !mbar_wait(&o_empty[s], ((k >> 1) - 1) & 1, a.status)) break;
        bool ok = true;
        for (int t = 0; t < ntiles; ++t, ++T) {
          const int sb = T % kNB;
          if (!mbar_wait(&v_ready[sb], (T / kNB) & 1, a.status)) { ok = false; break; }
          tc_fence_after();
          // A = P in TMEM (16 keys = 8 columns per step), B = V (MN-major: d
          // atoms KTC*128 bytes apart, 8-key groups 1 KB apart; 16 keys = 2 KB)
          const uint64_t dv = smem_desc(smem_u32(sV + sb * KV_BYTES), KTC * 128, 1024);
#pragma unroll
          for (int kk = 0; kk < KTC / 16; ++kk)
            mma_ts(tO0 + s * 128, tS + sb * KTC + kk * 8, smem_desc_at(dv, kk * 2048), kIdescO,
                    (t == 0 && kk == 0) ? 0u : 1u);
          mma_commit(&pv_done[sb]);
          mma_commit(&k_ready[sb]);  // S_{T+kNB} may start: the S/P buffer is free again
        }
        if (!ok) break;
      }
    }
    __syncwarp();
  } else if constexpr (BM == 64) {
    // ------------------------------------------------ softmax, M = 64 items
    // Item row m sits in TMEM lane 32 (m / 16) + m % 16, so lane quarter q
    // holds item rows 16q .. 16q + 15.  Warp w takes quarter w % 4 and half
    // w / 4 of every row's columns; with 16-lane accesses each thread holds two
    // rows (t / 4 and t / 4 + 8 of the quarter) x 16 columns of its half, and
    // the four threads t % 4 of a row finish its maxima and sums by shuffles.
    const int quarter = warp & 3, half = warp >> 2;
    const int cq = lane & 3;
    const int32_t rlA = quarter * 16 + (lane >> 2), rlB = rlA + 8;  // item rows of this thread
    const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
    auto xs = [&](int slot, int hf, int32_t rl) -> float& {
      return xch[(slot * 2 + hf) * kBM + rl];
    };
    auto pair_sync = [&]() { asm volatile("bar.sync %0, 64;" ::"r"(1 + quarter) : "memory"); };
    auto low = [](int32_t n) -> uint64_t {
      return n <= 0 ? 0ull : (n >= 64 ? ~0ull : ((1ull << n) - 1ull));
    };
    bool ok = true;
    uint32_t T = 0;
    for (int32_t k = 0; ok; ++k) {
      const int s = k & 1;
      if (!mbar_wait(&it_full[s], (k >> 1) & 1, a.status)) { ok = false; break; }
      const TcItem& it = items[s];
      const int32_t ntiles = it.ntiles;
      if (ntiles < 0) break;
      const int32_t b = it.b, g = it.g, split = it.split, row0 = it.row0;
      const int32_t rows_total = it.rows_total, cache = it.cache, Lk = it.Lk;
      const int32_t k_lo = it.k_lo, k_hi = it.k_hi;
      const bool direct = it.direct != 0;
      const int32_t* kflat = it.kflat;
      const uint32_t tO = tO0 + s * 128;
      const int32_t rA = row0 + rlA, rB = row0 + rlB;
      const bool liveA = rA < rows_total, liveB = rB < rows_total;
      const bool warp_live = row0 + quarter * 16 < rows_total;  // same for both warps of a pair
      const int32_t jqA = liveA ? rA / G : 0, hA = g * G + (liveA ? rA - jqA * G : 0);
      const int32_t jqB = liveB ? rB / G : 0, hB = g * G + (liveB ? rB - jqB * G : 0);
      const int32_t qposA = liveA ? kflat[jqA] : 0x7fffffff;
      const int32_t qposB = liveB ? kflat[jqB] : 0x7fffffff;
      const bool increasing = it.increasing != 0;
      int32_t minq = 0x7fffffff;
      const int32_t j_lo = row0 / G;
      if (increasing) {
        minq = kflat[j_lo];
      } else {
        const int32_t j_end = (min(rows_total, row0 + BM) + G - 1) / G;
        for (int32_t j = j_lo + lane; j < j_end; j += 32) minq = min(minq, kflat[j]);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) minq = min(minq, __shfl_xor_sync(0xffffffffu, minq, o));
      }
      const int32_t mask_from = min(cache, minq + 1);
      // visibility of the item's drafts to rows A and B (bit j: draft j visible)
      uint64_t vAlo = 0, vAhi = 0, vBlo = 0, vBhi = 0;
      if (warp_live && increasing) {
        const int32_t nA = jqA + 1, nB = jqB + 1;  // 1 .. 128
        vAlo = nA >= 64 ? ~0ull : ((1ull << nA) - 1ull);
        vAhi = nA <= 64 ? 0ull : (nA >= 128 ? ~0ull : ((1ull << (nA - 64)) - 1ull));
        vBlo = nB >= 64 ? ~0ull : ((1ull << nB) - 1ull);
        vBhi = nB <= 64 ? 0ull : (nB >= 128 ? ~0ull : ((1ull << (nB - 64)) - 1ull));
      } else if (warp_live) {
        const int32_t nd = Lk - cache;
#pragma unroll 1
        for (int j = 0; j < nd; j += 4) {
          const int4 kf = *reinterpret_cast<const int4*>(kflat + j);
          const uint64_t bA = (uint64_t)((uint32_t)(kf.x <= qposA) | ((uint32_t)(kf.y <= qposA) << 1) |
                                         ((uint32_t)(kf.z <= qposA) << 2) |
                                         ((uint32_t)(kf.w <= qposA) << 3));
          const uint64_t bB = (uint64_t)((uint32_t)(kf.x <= qposB) | ((uint32_t)(kf.y <= qposB) << 1) |
                                         ((uint32_t)(kf.z <= qposB) << 2) |
                                         ((uint32_t)(kf.w <= qposB) << 3));
          if (j < 64) {
            vAlo |= bA << j;
            vBlo |= bB << j;
          } else {
            vAhi |= bA << (j - 64);
            vBhi |= bB << (j - 64);
          }
        }
      }
      // keep mask of one row over keys c0 .. c0 + 63 (as in the M = 128 path)
      auto keep_of = [&](int32_t c0, int32_t qpos, uint64_t vlo, uint64_t vhi) -> uint64_t {
        const int32_t base = c0 - cache;  // draft index of column 0
        uint64_t win;
        if (base >= 128 || base <= -64) win = 0;
        else if (base >= 64) win = vhi >> (base - 64);
        else if (base > 0) win = (vlo >> base) | (vhi << (64 - base));
        else if (base == 0) win = vlo;
        else win = vlo << (-base);
        const int32_t seen_end = qpos < cache ? qpos + 1 : cache;
        return (low(seen_end - c0) | (win & ~low(cache - c0))) & low(k_hi - c0);
      };
      float m_runA = -INFINITY, m_runB = -INFINITY, l_runA = 0.f, l_runB = 0.f;
      for (int t = 0; t < ntiles; ++t, ++T) {
        const int bb = T & 1, sb = T % kNB;
        if (!mbar_wait(&s_full[sb], (T / kNB) & 1, a.status)) ok = false;
        tc_fence_after();
        float sv[32];
        if (warp_live) tld16x256_x8(tS + lane_off + sb * KTC + half * HC, sv);
        bool movedA = false, movedB = false;
        float alphaA = 1.f, alphaB = 1.f;
        uint32_t pk[16];
        if (warp_live) {
          const int32_t c0 = k_lo + t * KTC + half * HC;
          if (c0 + HC > k_hi || c0 + HC > mask_from) {
            const uint64_t keepA = keep_of(c0, qposA, vAlo, vAhi);
            const uint64_t keepB = keep_of(c0, qposB, vBlo, vBhi);
#pragma unroll
            for (int u = 0; u < 8; ++u)
#pragma unroll
              for (int e = 0; e < 2; ++e) {
                const int jj = 8 * u + 2 * cq + e;
                if (!((keepA >> jj) & 1ull)) sv[4 * u + e] = -INFINITY;
                if (!((keepB >> jj) & 1ull)) sv[4 * u + 2 + e] = -INFINITY;
              }
          }
          float a4[4], b4[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            a4[i] = fmaxf(fmaxf(sv[8 * i], sv[8 * i + 1]), fmaxf(sv[8 * i + 4], sv[8 * i + 5]));
            b4[i] = fmaxf(fmaxf(sv[8 * i + 2], sv[8 * i + 3]), fmaxf(sv[8 * i + 6], sv[8 * i + 7]));
          }
          float mxA = fmaxf(fmaxf(a4[0], a4[1]), fmaxf(a4[2], a4[3]));
          float mxB = fmaxf(fmaxf(b4[0], b4[1]), fmaxf(b4[2], b4[3]));
          mxA = fmaxf(mxA, __shfl_xor_sync(0xffffffffu, mxA, 1));
          mxB = fmaxf(mxB, __shfl_xor_sync(0xffffffffu, mxB, 1));
          mxA = fmaxf(mxA, __shfl_xor_sync(0xffffffffu, mxA, 2));
          mxB = fmaxf(mxB, __shfl_xor_sync(0xffffffffu, mxB, 2));
          // (the pair barrier also orders the partner's tcgen05.ld of S before
          // this warp overwrites the buffer with P)
          if (cq == 0) {
            xs(bb, half, rlA) = mxA;
            xs(bb, half, rlB) = mxB;
          }
          pair_sync();
          mxA = fmaxf(mxA, xs(bb, half ^ 1, rlA));
          mxB = fmaxf(mxB, xs(bb, half ^ 1, rlB));
          // move a running max only when it grows by more than 2^kRescale
          if (mxA != -INFINITY && (m_runA == -INFINITY || (mxA - m_runA) * c2 > kRescale)) {
            alphaA = (m_runA == -INFINITY) ? 0.f : ex2_approx((m_runA - mxA) * c2);
            m_runA = mxA;
            movedA = true;
          }
          if (mxB != -INFINITY && (m_runB == -INFINITY || (mxB - m_runB) * c2 > kRescale)) {
            alphaB = (m_runB == -INFINITY) ? 0.f : ex2_approx((m_runB - mxB) * c2);
            m_runB = mxB;
            movedB = true;
          }
          const float moffA = (m_runA == -INFINITY) ? 0.f : m_runA * c2;
          const float moffB = (m_runB == -INFINITY) ? 0.f : m_runB * c2;
          float sA[4] = {0.f, 0.f, 0.f, 0.f}, sB[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
          for (int u = 0; u < 8; ++u) {
            const float eA0 = ex2_approx(fmaf(sv[4 * u], c2, -moffA));
            const float eA1 = ex2_approx(fmaf(sv[4 * u + 1], c2, -moffA));
            const float eB0 = ex2_approx(fmaf(sv[4 * u + 2], c2, -moffB));
            const float eB1 = ex2_approx(fmaf(sv[4 * u + 3], c2, -moffB));
            sA[u & 3] += eA0 + eA1;
            sB[u & 3] += eB0 + eB1;
            pk[2 * u] = pack_bf16x2(eA0, eA1);
            pk[2 * u + 1] = pack_bf16x2(eB0, eB1);
          }
          l_runA = l_runA * alphaA + ((sA[0] + sA[1]) + (sA[2] + sA[3]));
          l_runB = l_runB * alphaB + ((sB[0] + sB[1]) + (sB[2] + sB[3]));
        }
        if (warp_live) {
          // O may be rescaled once PV_{T-1} is done
          if (__any_sync(0xffffffffu, (movedA || movedB) && t > 0)) {
            if (!mbar_wait(&pv_done[(T - 1) % kNB], ((T - 1) / kNB) & 1, a.status)) ok = false;
            tc_fence_after();
            float ov[HD / 2];
            const uint32_t ta = tO + lane_off + half * HD;
            if constexpr (HD == 64) tld16x256_x8(ta, ov);
            else tld16x256_x4(ta, ov);
#pragma unroll
            for (int u = 0; u < HD / 8; ++u) {
              ov[4 * u] *= alphaA;
              ov[4 * u + 1] *= alphaA;
              ov[4 * u + 2] *= alphaB;
              ov[4 * u + 3] *= alphaB;
            }
            if constexpr (HD == 64) tst16x256_x8(ta, ov);
            else tst16x256_x4(ta, ov);
          }
          // P_T as bf16 pairs over the first half of its S buffer: this half's
          // keys are word columns [half * HC / 2, (half + 1) * HC / 2)
          tst16x128_x8(tS + lane_off + sb * KTC + half * (HC / 2), pk);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&v_ready[sb]);
      }
      // ---- epilogue: wait for the item's last PV product, normalise, write this half
      const uint32_t Tl = T - 1;
      if (!mbar_wait(&pv_done[Tl % kNB], (Tl / kNB) & 1, a.status)) ok = false;
      tc_fence_after();
      if (warp_live) {
        float lA = l_runA, lB = l_runB;
        lA += __shfl_xor_sync(0xffffffffu, lA, 1);
        lB += __shfl_xor_sync(0xffffffffu, lB, 1);
        lA += __shfl_xor_sync(0xffffffffu, lA, 2);
        lB += __shfl_xor_sync(0xffffffffu, lB, 2);
        if (cq == 0) {
          xs(2, half, rlA) = lA;
          xs(2, half, rlB) = lB;
        }
        pair_sync();
        const float ltA = lA + xs(2, half ^ 1, rlA), ltB = lB + xs(2, half ^ 1, rlB);
        const float invA = ltA > 0.f ? __fdividef(1.0f, ltA) : 0.f;
        const float invB = ltB > 0.f ? __fdividef(1.0f, ltB) : 0.f;
        float ov[HD / 2];
        const uint32_t ta = tO + lane_off + half * HD;
        if constexpr (HD == 64) tld16x256_x8(ta, ov);
        else tld16x256_x4(ta, ov);
        // (debug builds: the rows' store indexes against their buffers)
        const int64_t n_rows_o = (int64_t)a.B * a.D_max * a.Hq;
        const int64_t n_rows_p = (int64_t)a.B * a.Hq * a.D_max * L.splits;
        const bool sA = liveA && (direct ? dbg_in(((int64_t)b * a.D_max + jqA) * a.Hq + hA, n_rows_o, a.status)
                                         : dbg_in((((int64_t)b * a.Hq + hA) * a.D_max + jqA) * L.splits + split, n_rows_p, a.status));
        const bool sB = liveB && (direct ? dbg_in(((int64_t)b * a.D_max + jqB) * a.Hq + hB, n_rows_o, a.status)
                                         : dbg_in((((int64_t)b * a.Hq + hB) * a.D_max + jqB) * L.splits + split, n_rows_p, a.status));
        if (ok) {
          const int colb = half * HD + 2 * cq;
          if (direct) {
            __nv_bfloat16* oA = reinterpret_cast<__nv_bfloat16*>(a.o) +
                                (((int64_t)b * a.D_max + jqA) * a.Hq + hA) * D + colb;
            __nv_bfloat16* oB = reinterpret_cast<__nv_bfloat16*>(a.o) +
                                (((int64_t)b * a.D_max + jqB) * a.Hq + hB) * D + colb;
#pragma unroll
            for (int u = 0; u < HD / 8; ++u) {
              if (sA)
                *reinterpret_cast<uint32_t*>(oA + 8 * u) =
                    pack_bf16x2(ov[4 * u] * invA, ov[4 * u + 1] * invA);
              if (sB)
                *reinterpret_cast<uint32_t*>(oB + 8 * u) =
                    pack_bf16x2(ov[4 * u + 2] * invB, ov[4 * u + 3] * invB);
            }
          } else {
            float* pA = L.part_o +
                        ((((int64_t)b * a.Hq + hA) * a.D_max + jqA) * L.splits + split) * D + colb;
            float* pB = L.part_o +
                        ((((int64_t)b * a.Hq + hB) * a.D_max + jqB) * L.splits + split) * D + colb;
#pragma unroll
            for (int u = 0; u < HD / 8; ++u) {
              if (sA)
                *reinterpret_cast<float2*>(pA + 8 * u) =
                    make_float2(ov[4 * u] * invA, ov[4 * u + 1] * invA);
              if (sB)
                *reinterpret_cast<float2*>(pB + 8 * u) =
                    make_float2(ov[4 * u + 2] * invB, ov[4 * u + 3] * invB);
            }
          }
          if (half == 0 && cq == 0) {
            const float lseA =
                ltA > 0.f ? (m_runA * (c2 / kLog2eTC) + __logf(ltA)) : -INFINITY;
            const float lseB =
                ltB > 0.f ? (m_runB * (c2 / kLog2eTC) + __logf(ltB)) : -INFINITY;
            if (direct) {
              if (a.lse != nullptr && sA) a.lse[((int64_t)b * a.Hq + hA) * a.D_max + jqA] = lseA;
              if (a.lse != nullptr && sB) a.lse[((int64_t)b * a.Hq + hB) * a.D_max + jqB] = lseB;
            } else {
              if (sA)
                L.part_lse[(((int64_t)b * a.Hq + hA) * a.D_max + jqA) * L.splits + split] = lseA;
              if (sB)
                L.part_lse[(((int64_t)b * a.Hq + hB) * a.D_max + jqB) * L.splits + split] = lseB;
            }
          }
        }
      }
      // O[s] and the item slot are free for item k + 2
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&o_empty[s]);
        mbar_arrive(&it_empty[s]);
      }
    }
  } else {
    // ------------------------------------------------------------- softmax
    const int quarter = warp & 3, half = warp >> 2;
    const int32_t rl = quarter * 32 + lane;   // row inside the tile = TMEM lane
    const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
    // partial values of the two halves of a row: slots 0 / 1 by tile parity, 2 for the epilogue
    auto xslot = [&](int slot, int hf) -> float& { return xch[(slot * 2 + hf) * kBM + rl]; };
    auto pair_sync = [&]() { asm volatile("bar.sync %0, 64;" ::"r"(1 + quarter) : "memory"); };
    bool ok = true;
    uint32_t T = 0;
    for (int32_t k = 0; ok; ++k) {
      const int s = k & 1;
      if (!mbar_wait(&it_full[s], (k >> 1) & 1, a.status)) { ok = false; break; }
      const TcItem& it = items[s];
      const int32_t ntiles = it.ntiles;
      if (ntiles < 0) break;
      const int32_t b = it.b, g = it.g, split = it.split, row0 = it.row0;
      const int32_t rows_total = it.rows_total, cache = it.cache, Lk = it.Lk;
      const int32_t k_lo = it.k_lo, k_hi = it.k_hi;
      const bool direct = it.direct != 0;
      const int32_t* kflat = it.kflat;
      const uint32_t tO = tO0 + s * 128;
      const int32_t r = row0 + rl;              // this thread's query row
      const bool live = r < rows_total;
      const bool warp_live = row0 + quarter * 32 < rows_total;  // same for both warps of a pair
      // this row's draft and query head (computed once per item)
      const int32_t jq = live ? r / G : 0, h = g * G + (live ? r - (r / G) * G : 0);
      const int32_t qpos = live ? kflat[jq] : 0x7fffffff;
      const bool increasing = it.increasing != 0;
      // cache slots below every query position of this item are visible to all rows
      int32_t minq = 0x7fffffff;
      const int32_t j_lo = row0 / G;
      if (increasing) {
        minq = kflat[j_lo];
      } else {
        const int32_t j_end = (min(rows_total, row0 + kBM) + G - 1) / G;
        for (int32_t j = j_lo + lane; j < j_end; j += 32) minq = min(minq, kflat[j]);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) minq = min(minq, __shfl_xor_sync(0xffffffffu, minq, o));
      }
      const int32_t mask_from = min(cache, minq + 1);
      // visibility of the item's drafts to this row: bit j of (vis_hi:vis_lo) is
      // kflat[j] <= qpos, that is j <= jq for increasing positions.  Runs once
      // per item, so the general loop is kept rolled (small code: a cold
      // unrolled path costs instruction-cache misses).
      uint64_t vis_lo = 0, vis_hi = 0;
      if (warp_live && increasing) {
        const int32_t n = jq + 1;  // 1 .. 128
        vis_lo = n >= 64 ? ~0ull : ((1ull << n) - 1ull);
        vis_hi = n <= 64 ? 0ull : (n >= 128 ? ~0ull : ((1ull << (n - 64)) - 1ull));
      } else if (warp_live) {
        const int32_t nd = Lk - cache;
#pragma unroll 1
        for (int j = 0; j < nd; j += 4) {
          const int4 kf = *reinterpret_cast<const int4*>(kflat + j);
          const uint64_t bits = (uint64_t)((uint32_t)(kf.x <= qpos) | ((uint32_t)(kf.y <= qpos) << 1) |
                                           ((uint32_t)(kf.z <= qpos) << 2) |
                                           ((uint32_t)(kf.w <= qpos) << 3));
          if (j < 64) vis_lo |= bits << j;
          else vis_hi |= bits << (j - 64);
        }
      }
      float m_run = -INFINITY, l_run = 0.f;  // l_run: this half's partial sum
      for (int t = 0; t < ntiles; ++t, ++T) {
        const int bb = T & 1, sb = T % kNB;
        if (!mbar_wait(&s_full[sb], (T / kNB) & 1, a.status)) ok = false;
        tc_fence_after();
        float sv[HC];
        if (warp_live) {
          tmem_ld32(tS + lane_off + sb * KTC + half * HC, sv);
          tmem_ld32(tS + lane_off + sb * KTC + half * HC + 32, sv + 32);
        }
        bool moved = false;
        float alpha = 1.f;
        uint32_t pk[HC / 2];
        if (warp_live) {
          // mask: keys past this split / the sequence, and the spatial predicate
          const int32_t c0 = k_lo + t * KTC + half * HC;
          if (c0 + HC > k_hi || c0 + HC > mask_from) {
            // keep bit jj: key c0 + jj is visible to this row.  Cache keys are a
            // prefix of the window (visible up to qpos), draft keys come from the
            // visibility bits, keys past the split are dropped.
            auto low = [](int32_t n) -> uint64_t {
              return n <= 0 ? 0ull : (n >= 64 ? ~0ull : ((1ull << n) - 1ull));
            };
            const int32_t base = c0 - cache;  // draft index of column 0
            uint64_t win;                     // bit jj: draft base + jj is visible
            if (base >= 128 || base <= -64) win = 0;
            else if (base >= 64) win = vis_hi >> (base - 64);
            else if (base > 0) win = (vis_lo >> base) | (vis_hi << (64 - base));
            else if (base == 0) win = vis_lo;
            else win = vis_lo << (-base);
            const int32_t seen_end = qpos < cache ? qpos + 1 : cache;
            const uint64_t keep =
                (low(seen_end - c0) | (win & ~low(cache - c0))) & low(k_hi - c0);
#pragma unroll
            for (int jj = 0; jj < HC; ++jj)
              if (!((keep >> jj) & 1ull)) sv[jj] = -INFINITY;
          }
          // tree reductions: short dependency chains
          float m8[HC / 4];
#pragma unroll
          for (int i = 0; i < HC / 4; ++i)
            m8[i] = fmaxf(fmaxf(sv[4 * i], sv[4 * i + 1]), fmaxf(sv[4 * i + 2], sv[4 * i + 3]));
#pragma unroll
          for (int w = HC / 8; w >= 1; w >>= 1)
#pragma unroll
            for (int i = 0; i < w; ++i) m8[i] = fmaxf(m8[i], m8[i + w]);
          float mx = m8[0];
          // (the pair barrier also orders the partner's tcgen05.ld of S before
          // this warp overwrites the buffer with P)
          xslot(bb, half) = mx;
          pair_sync();
          mx = fmaxf(mx, xslot(bb, half ^ 1));
          // move the running max only when it grows by more than 2^kRescale
          if (mx != -INFINITY && (m_run == -INFINITY || (mx - m_run) * c2 > kRescale)) {
            alpha = (m_run == -INFINITY) ? 0.f : ex2_approx((m_run - mx) * c2);
            m_run = mx;
            moved = true;
          }
          const float moff = (m_run == -INFINITY) ? 0.f : m_run * c2;
          float r8[HC / 4];
#pragma unroll
          for (int i = 0; i < HC / 4; ++i) {
            const float e0 = ex2_approx(fmaf(sv[4 * i], c2, -moff));
            const float e1 = ex2_approx(fmaf(sv[4 * i + 1], c2, -moff));
            const float e2 = ex2_approx(fmaf(sv[4 * i + 2], c2, -moff));
            const float e3 = ex2_approx(fmaf(sv[4 * i + 3], c2, -moff));
            r8[i] = (e0 + e1) + (e2 + e3);
            pk[2 * i] = pack_bf16x2(e0, e1);
            pk[2 * i + 1] = pack_bf16x2(e2, e3);
          }
#pragma unroll
          for (int w = HC / 8; w >= 1; w >>= 1)
#pragma unroll
            for (int i = 0; i < w; ++i) r8[i] += r8[i + w];
          l_run = l_run * alpha + r8[0];
        }
        // O may be rescaled once PV_{T-1} is done
        if (warp_live) {
          if (__any_sync(0xffffffffu, moved && t > 0)) {
            if (!mbar_wait(&pv_done[(T - 1) % kNB], ((T - 1) / kNB) & 1, a.status)) ok = false;
            tc_fence_after();
            float ov[32];
#pragma unroll 1
            for (int cc = 0; cc < HD / 32; ++cc) {
              const uint32_t ta = tO + lane_off + half * HD + cc * 32;
              tmem_ld32(ta, ov);
#pragma unroll
              for (int i = 0; i < 32; ++i) ov[i] *= alpha;
              tmem_st32(ta, ov);
            }
          }
          // P_T as bf16 pairs over the first half of its S buffer: this half's keys
          // are columns [half * HC / 2, (half + 1) * HC / 2)
          tmem_st32(tS + lane_off + sb * KTC + half * (HC / 2), pk);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&v_ready[sb]);
      }
      // ---- epilogue: wait for the item's last PV product, normalise, write this half
      const uint32_t Tl = T - 1;
      if (!mbar_wait(&pv_done[Tl % kNB], (Tl / kNB) & 1, a.status)) ok = false;
      tc_fence_after();
      if (warp_live) {
        xslot(2, half) = l_run;
        pair_sync();
        const float l_tot = l_run + xslot(2, half ^ 1);
        // fast reciprocal and logarithm: the epilogue runs once per item, and
        // its instruction count is its cost
        const float inv_l = l_tot > 0.f ? __fdividef(1.0f, l_tot) : 0.f;
        const float lse = (l_tot > 0.f) ? (m_run * (c2 / kLog2eTC) + __logf(l_tot)) : -INFINITY;
        // (debug builds: the row's store index against its buffer)
        const bool sL = live && (direct ? dbg_in(((int64_t)b * a.D_max + jq) * a.Hq + h,
                                                 (int64_t)a.B * a.D_max * a.Hq, a.status)
                                        : dbg_in((((int64_t)b * a.Hq + h) * a.D_max + jq) * L.splits + split,
                                                 (int64_t)a.B * a.Hq * a.D_max * L.splits, a.status));
#pragma unroll 1
        for (int cc = 0; cc < HD / 32; ++cc) {
          float ov[32];
          tmem_ld32(tO + lane_off + half * HD + cc * 32, ov);
          if (!sL || !ok) continue;
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
              *reinterpret_cast<float4*>(po + i) = make_float4(
                  ov[i] * inv_l, ov[i + 1] * inv_l, ov[i + 2] * inv_l, ov[i + 3] * inv_l);
          }
        }
        if (sL && ok && half == 0) {
          if (direct) {
            if (a.lse != nullptr) a.lse[((int64_t)b * a.Hq + h) * a.D_max + jq] = lse;
          } else {
            L.part_lse[(((int64_t)b * a.Hq + h) * a.D_max + jq) * L.splits + split] = lse;
          }
        }
      }
      // O[s] and the item slot are free for item k + 2
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&o_empty[s]);
        mbar_arrive(&it_empty[s]);
      }
    }
  }
  // ---- teardown
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

}  // namespace

#ifndef SSD_ATTN_TC_MIN_ROWS
#define SSD_ATTN_TC_MIN_ROWS 16  // query rows per KV group above which the tcgen05 kernel runs
#endif

bool attention_tc_supported(int32_t Hq, int32_t Hkv, int32_t d, int32_t D_max) {
  const int32_t G = Hq / Hkv;
  return (d == 64 || d == 128) && G >= 1 && G <= kBM && (kBM % G) == 0 &&
         D_max * G > SSD_ATTN_TC_MIN_ROWS;
}

namespace {
// Query rows per tile: 64 when a KV group's rows fit (M = 64 products, their
// softmax spread over the four lane quarters), else 128.
int32_t tc_tile_rows(int32_t D_max, int32_t G) { return D_max * G <= 64 ? 64 : kBM; }
}  // namespace

TcPlan attention_tc_plan(int32_t B, int32_t Hq, int32_t Hkv, int32_t D_max, int32_t L_max) {
  TcPlan p;
  const int32_t G = Hq / Hkv;
  const int32_t bm = tc_tile_rows(D_max, G);
  p.mtiles = (D_max * G + bm - 1) / bm;
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
                                float* part_lse, cudaStream_t stream, bool pdl) {
  EncodeTiledFn fn = tensor_map_encoder();
  if (fn == nullptr) return cudaErrorInvalidValue;
  const int32_t G = a.Hq / a.Hkv;
  const int32_t bm = tc_tile_rows(a.D_max, G);
  CUtensorMap tq, tk, tv;
  {
    cuuint64_t dims[3] = {(cuuint64_t)a.d, (cuuint64_t)a.Hq, (cuuint64_t)a.B * a.D_max};
    cuuint64_t strides[2] = {(cuuint64_t)a.d * 2, (cuuint64_t)a.Hq * a.d * 2};
    cuuint32_t box[3] = {64, (cuuint32_t)G, (cuuint32_t)(bm / G)};
    cuuint32_t estr[3] = {1, 1, 1};
    if (fn(&tq, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(a.q), dims, strides, box,
           estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  const int64_t rows = (int64_t)a.B * a.Hkv * a.L_max;
  for (int w = 0; w < 2; ++w) {
    // d = 128: {64 columns, rows, 2 halves}, the halves 128 B apart inside a row,
    // so one box {64, KTC, 2} is a whole tile; d = 64: {64, rows}, box {64, KTC}
    const cuuint32_t rank = a.d == 128 ? 3 : 2;
    cuuint64_t dims[3] = {64, (cuuint64_t)rows, 2};
    cuuint64_t strides[2] = {(cuuint64_t)a.d * 2, 128};
    cuuint32_t box[3] = {64, KTC, 2};
    cuuint32_t estr[3] = {1, 1, 1};
    if (fn(w == 0 ? &tk : &tv, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank,
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
  // persistent: one CTA per SM (at most one per work item)
  const int64_t n_items = (int64_t)a.B * a.Hkv * p.mtiles * p.splits;
  const dim3 grid((unsigned)std::min<int64_t>(n_items, device_sm_count()));
  const dim3 block(kThreadsTC);
  auto launch = [&](auto kernel, size_t smem) {
    cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    return launch_kernel(kernel, grid, block, smem, stream, pdl, tq, tk, tv, a, L);
  };
  if (a.d == 128)
    return bm == 64 ? launch(frontier_attn_tc_kernel<128, 64>, tc_smem_bytes<128, 64>())
                    : launch(frontier_attn_tc_kernel<128, 128>, tc_smem_bytes<128, 128>());
  return bm == 64 ? launch(frontier_attn_tc_kernel<64, 64>, tc_smem_bytes<64, 64>())
                  : launch(frontier_attn_tc_kernel<64, 128>, tc_smem_bytes<64, 128>());
}

}  // namespace ssd
