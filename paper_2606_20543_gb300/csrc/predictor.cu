// predictor.cu — the spatial draft predictor f_phi (Sec. 3.3 "Draft
// Prediction in Latent Space", Eq. 2) and the draft tokens it yields:
//
//   h_hat = W0 z + SwiGLU(RMSNorm(W0 z)),  z = [h ; e],
//   SwiGLU(x) = W2 (silu(W1 x) * W3 x),    t_hat = argmax GenHead(RMSNorm(h_hat)).
//
// Design (GB300): for one grid row of positions the predictor is a chain of
// skinny products — at most 128 rows against four weight matrices of 64 MB
// and the 128 MB GenHead at the paper's head size — so it is bound by reading
// the weights once from HBM.  One persistent cooperative kernel (one CTA per
// SM) runs the whole chain in four phases.  RMSNorm(x) g = s(x) (x * g) with
// the row scale s(x) = 1 / sqrt(mean(x^2) + eps), and s commutes with the
// products that follow, so every product input is an elementwise bf16 array
// that the previous phase writes tile by tile, and the row scale is applied
// to the product's output:
//   P0  A  = W0 z                        (features d, K = 2d);  Ag = bf16(A * g1)
//   P1  U  = s(A) W1 Ag, Vg = s(A) W3 Ag (features m, K = d);   G = bf16(silu(U) * Vg)
//   P2  h  = A + W2 G                    (features d, K = m);   Hg = bf16(h * g2)
//   P3  l  = W_head^T Hg                 (features V, K = d);   t = argmax l
// (the GenHead's row scale s(h) > 0 leaves the argmax unchanged; the lowest
// index wins ties).  Every product is D[128 features x N rows] += W[128 x 16]
// X[16 x N] on the tensor cores (tcgen05.mma kind::f16, fp32 accumulation in
// tensor memory): weights on M, the rows (padded to N, a multiple of 16) on N.
// A phase's work is a list of units (128 features x 128 K, or 128 features x
// 64 K of both W1 and W3), 32 KB of weights each; CTA c takes one contiguous
// range of every phase's units, so a feature tile is split over at most a few
// CTAs along K (split-K partials summed in a fixed order).
//   * warps 0, 1: weight producers (alternate units, one or two TMA copies per
//     unit) running ahead through all four phases: the weights do not depend
//     on the activations, so the weight stream keeps going while a phase
//     waits for the previous one to finish;
//   * warp 3: activation producer — lane 0 issues one TMA copy of each
//     unit's activation tile X (K-major, 128-byte swizzle) from z, Ag, G or
//     Hg once the tile of the previous phase that X is cut from is final.
//     With at most 80 rows the unit waits for that one tile (the whole warp
//     polls a window of 32 tiles per round trip, so a CTA starts a phase as
//     soon as the tiles it reads are final, not the last tile of the grid);
//     with more rows, where a tile's finish is heavier and competes with the
//     next phase's stream, for every tile of the previous phase.  Warp 3 also
//     allocates and frees the tensor memory;
//   * warp 2: issues the MMAs of each unit into one of two TMEM accumulators
//     (the next tile's products overlap the previous tile's epilogue);
//   * warps 4-7: the epilogue.  Each TMEM lane is one feature; the CTA's
//     partial of a tile goes to the workspace (even and odd phases in
//     separate buffers, since a CTA may start a phase while another still sums
//     the previous phase's partials), then a ticket per tile: the last
//     contributor sums the tile's partials in slot order and finishes it (A,
//     Ag and A's squares per row; G; h and Hg; the tile's argmax per row,
//     raised into one 64-bit key per row by a max reduction), then counts the
//     tile final on its ticket and on the phase's counter.  The row scales
//     s(A) are summed once per CTA from the P0 tiles' squares before its first
//     P1 finish; the last tile of P3 to finish turns the keys into the tokens.
// Numerics: every product input is bf16 (z, the weights, Ag, G, Hg); A, U,
// Vg, h and the logits are fp32; every sum runs in a fixed order, so results
// do not depend on timing.
#include <algorithm>

#include "kernels.cuh"

namespace ssd {

namespace {

constexpr int kPThreads = 256;       // 8 warps
constexpr int kWarpMma = 2;
constexpr int kWarpX = 3;            // activation producer; allocates / frees tensor memory
constexpr int kEpiWarp0 = 4;         // warps 4-7: TMEM lane quarters 0-3
constexpr int kEpiThreads = 128;
constexpr int kUnitBytes = 32768;    // weights per unit
constexpr int kMaxRows = 128;
constexpr int kPhases = 4;
constexpr int kBarEpi = 1;           // named barrier of the epilogue warps
constexpr int kMaxSlots = 8;         // most CTAs sharing one feature tile
constexpr int kTileWaitRows = 80;    // up to this many rows: per-tile activation waits
// One 128-byte line per row's argmax key: every GenHead tile raises every
// row's key near the end of the kernel, and the rows' reductions go to
// separate lines.
constexpr int kKeyStride = 16;

struct PredPhase {
  int32_t units;    // units of the phase
  int32_t upt;      // units per feature tile
  int32_t tiles;    // feature tiles of 128
  int32_t kw;       // K per unit: 128, or 64 (P1: W1 and W3 tiles of 64)
  int32_t slots;    // most CTAs contributing to one tile
};

struct PredLaunch {
  PredPhase ph[kPhases];
  int32_t ncta, rows, nn, nc;  // rows, MMA N (rows padded to 16), TMEM columns per accumulator
  int32_t stages;              // ring slots (weights + activations of one unit each)
  int32_t d, m, V;
  uint32_t max_polls, shortfall;
  int32_t tile_waits;          // activation copies wait per tile (else per phase)
  float eps;
  const float* gamma1;
  const float* gamma2;
  float* hid;                  // fp32 [rows][d]: A, then h_hat
  __nv_bfloat16* ag;           // bf16 [rows][d]: A * g1, then h_hat * g2
  __nv_bfloat16* g;            // bf16 [rows][m]: silu(U) * Vg
  float* ss;                   // fp32 [d/128][128]: per-tile sums of squares of A's rows
  unsigned long long* best;    // [rows][kKeyStride]: the argmax key of row r at best[r * kKeyStride]
  float* part;                 // split-K partials: even phases at part, odd at part + part_odd
  int64_t part_odd;
  unsigned int* ctr;           // tickets [4][max tiles], done [4], abort
  int32_t max_tiles;
  int32_t* out_tok;
  int32_t* status;
};

__device__ __forceinline__ int64_t unit_start(int32_t c, int32_t units, int32_t ncta) {
  return (int64_t)c * units / ncta;
}
// The CTA whose range holds unit u.
__device__ __forceinline__ int32_t unit_cta(int64_t u, int32_t units, int32_t ncta) {
  return (int32_t)(((u + 1) * ncta + units - 1) / units) - 1;
}

__device__ __forceinline__ void bar_named(int id, int count) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}

// Named barrier that also ORs a predicate over its `count` threads: every
// thread of the group leaves with the same answer from the same barrier.
__device__ __forceinline__ bool bar_or(int id, int count, bool pred) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n"
      " bar.red.or.pred q, %2, %3, p;\n selp.u32 %0, 1, 0, q;\n}\n"
      : "=r"(r)
      : "r"(pred ? 1u : 0u), "r"(id), "r"(count)
      : "memory");
  return r != 0;
}

__device__ __forceinline__ uint32_t ld_acquire_u32(const unsigned int* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Order this thread's generic-proxy global accesses with async-proxy (TMA)
// accesses: after writing an array that other CTAs will load by TMA, and
// after learning that such an array is complete, before loading it.
__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

// Release / acquire at GPU scope (lighter than a sequentially consistent
// fence): orders this thread's earlier writes before, and its later reads
// after, the ticket and counter atomics that publish and claim them.
__device__ __forceinline__ void fence_acq_rel_gpu() {
  asm volatile("fence.acq_rel.gpu;" ::: "memory");
}

// Counters, one per 128-byte line so that CTAs counting different tiles do
// not contend for one line: tickets [4][max tiles], done [4], abort.
constexpr int kCtrStride = 32;
__device__ __forceinline__ unsigned int* ticket(const PredLaunch& L, int p, int f) {
  return L.ctr + (p * L.max_tiles + f) * kCtrStride;
}
__device__ __forceinline__ unsigned int* done_ctr(const PredLaunch& L, int p) {
  return L.ctr + (kPhases * L.max_tiles + p) * kCtrStride;
}
__device__ __forceinline__ unsigned int* abort_flag(const PredLaunch& L) {
  return L.ctr + (kPhases * L.max_tiles + kPhases) * kCtrStride;
}

// Bounded wait until *ctr >= target; false (SSD_ERR_TIMEOUT recorded, abort
// raised) if it gave up, or if another CTA aborted the kernel.
__device__ bool wait_count(const PredLaunch& L, const unsigned int* ctr, uint32_t target) {
  for (uint32_t i = 0; i < L.max_polls; ++i) {
    if (ld_acquire_u32(ctr) >= target) return ld_acquire_u32(abort_flag(L)) == 0u;
    if ((i & 1023u) == 1023u && ld_acquire_u32(abort_flag(L)) != 0u) return false;
    if (i > 64) __nanosleep(128);
  }
  atomicExch(abort_flag(L), 1u);
  record_status(L.status, SSD_ERR_TIMEOUT);
  return false;
}

__device__ __forceinline__ void warp_argmax(float& v, int32_t& i) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, v, o);
    const int32_t oi = __shfl_xor_sync(0xffffffffu, i, o);
    if (ov > v || (ov == v && oi < i)) {
      v = ov;
      i = oi;
    }
  }
}

}  // namespace

namespace {

// The vocabulary argmax of each row is kept as one 64-bit key per row,
// raised by a max reduction from every finished GenHead tile: the logit in an
// order-preserving unsigned form (NaN as the lowest key) above the inverted
// index, so the largest logit wins and the lower index among equal ones
// (-0 is taken as +0, which compares equal to it).
__device__ __forceinline__ unsigned long long argmax_key(float v, int32_t i) {
  uint32_t u = v == 0.f ? 0u : __float_as_uint(v);
  u = (v != v) ? 0u : ((u & 0x80000000u) ? ~u : (u | 0x80000000u));
  return ((unsigned long long)u << 32) | (unsigned long long)(0xffffffffu - (uint32_t)i);
}
__device__ __forceinline__ int32_t argmax_index(unsigned long long key) {
  return (int32_t)(0xffffffffu - (uint32_t)(key & 0xffffffffull));
}

// The finishing step of one row r of a tile from its summed products x.
// P0 (p = 0): A = x, Ag = bf16(A * g1) and A's squares; P2: h = A + x,
// Hg = bf16(h * g2).
__device__ __forceinline__ void emit_hidden(const PredLaunch& L, int p, int32_t f, int32_t r,
                                            int32_t feat, int q, float4 x, float4 a0, float4 ga) {
  float4 y = x;
  if (p == 2) y = make_float4(a0.x + y.x, a0.y + y.y, a0.z + y.z, a0.w + y.w);
  *reinterpret_cast<float4*>(L.hid + (int64_t)r * L.d + feat) = y;
  uint2 o;
  o.x = pack_bf16x2(y.x * ga.x, y.y * ga.y);
  o.y = pack_bf16x2(y.z * ga.z, y.w * ga.w);
  *reinterpret_cast<uint2*>(L.ag + (int64_t)r * L.d + feat) = o;
  if (p == 0) {
    const float sq = warp_sum((y.x * y.x + y.y * y.y) + (y.z * y.z + y.w * y.w));
    if (q == 0) L.ss[(int64_t)f * 128 + r] = sq;
  }
}
// P1: G = bf16(silu(U) * Vg) with U, Vg scaled by the row's s(A).
__device__ __forceinline__ void emit_gate(const PredLaunch& L, int32_t r, int32_t feat, float4 uu,
                                          float4 vv, float sr) {
  const float u0 = uu.x * sr, u1 = uu.y * sr, u2 = uu.z * sr, u3 = uu.w * sr;
  uint2 o;
  o.x = pack_bf16x2(u0 / (1.0f + expf(-u0)) * (vv.x * sr), u1 / (1.0f + expf(-u1)) * (vv.y * sr));
  o.y = pack_bf16x2(u2 / (1.0f + expf(-u2)) * (vv.z * sr), u3 / (1.0f + expf(-u3)) * (vv.w * sr));
  *reinterpret_cast<uint2*>(L.g + (int64_t)r * L.m + feat) = o;
}
// P3: the tile's argmax for row r (lowest index on ties) raised into the row's key.
__device__ __forceinline__ void emit_argmax(const PredLaunch& L, int32_t r, int32_t feat, int q,
                                            float4 x) {
  float bv = x.x;
  int32_t bi = feat;
  if (x.y > bv) { bv = x.y; bi = feat + 1; }
  if (x.z > bv) { bv = x.z; bi = feat + 2; }
  if (x.w > bv) { bv = x.w; bi = feat + 3; }
  warp_argmax(bv, bi);
  if (q == 0) {  // a reduction without a result: the warp goes on at once (measured:
                 // atomicMax here held each row's finish for a round trip)
    const unsigned long long key = argmax_key(bv, bi);
    asm volatile("red.relaxed.gpu.global.max.u64 [%0], %1;"
                 ::"l"(L.best + (int64_t)r * kKeyStride), "l"(key) : "memory");
  }
}

// Epilogue of the last contributor of tile f of phase p: the tile's partials
// summed in slot order, then the phase's finishing step.  Thread et (0..127)
// takes features f * 128 + 4 q .. + 3 (q = et % 32, 16-byte loads) of rows
// et / 32 + 4 i; the 32 lanes of a warp hold one row's 128 features, so row
// reductions are warp reductions.  Each batch issues RB rows x NACC
// accumulators x SMAX slots (at most 32 float4) before summing any, so a tile
// costs a few round trips to L2.  srow: [128] the row scales s(A) (P1).
template <int SMAX, int NACC>
__device__ void finish_tile_t(const PredLaunch& L, int p, int32_t f, int32_t cnt, int et,
                              const float* srow) {
  // rows per batch: up to 32 loads in flight, at most 8 rows (a longer unrolled
  // body only lengthens code that runs once per phase; 8 rows cover 24-row
  // calls in one batch)
  constexpr int RB = 32 / (SMAX * NACC) > 8 ? 8 : (32 / (SMAX * NACC) > 0 ? 32 / (SMAX * NACC) : 1);
  const PredPhase& ph = L.ph[p];
  const int w = et >> 5, q = et & 31;
  const int32_t feat = f * 128 + 4 * q;
  const int64_t tile_stride = (int64_t)NACC * L.nn * 128;
  const float* base = L.part + (p & 1) * L.part_odd + (int64_t)f * ph.slots * tile_stride + 4 * q;
  float4 ga = make_float4(0.f, 0.f, 0.f, 0.f);
  if (p == 0) ga = __ldg(reinterpret_cast<const float4*>(L.gamma1 + feat));
  if (p == 2) ga = __ldg(reinterpret_cast<const float4*>(L.gamma2 + feat));
  const int32_t my_rows = (L.rows - w + 3) / 4;
  for (int32_t i0 = 0; i0 < my_rows; i0 += RB) {
    float4 v[RB][NACC][SMAX];
#pragma unroll
    for (int b = 0; b < RB; ++b)
#pragma unroll
      for (int a = 0; a < NACC; ++a)
#pragma unroll
        for (int sl = 0; sl < SMAX; ++sl) {
          v[b][a][sl] = make_float4(0.f, 0.f, 0.f, 0.f);
          if (sl < cnt && i0 + b < my_rows) {
            const int32_t r = w + 4 * (i0 + b);
            v[b][a][sl] = __ldcg(reinterpret_cast<const float4*>(
                base + sl * tile_stride + ((int64_t)a * L.nn + r) * 128));
          }
        }
    // each row's sums (and, in P2, its A) first, all loads in flight; then
    // one rolled loop finishes the rows, so that the finishing code exists
    // once in the instruction stream.  It runs once per phase, and between
    // calls other kernels evict it: an unrolled copy per row was fetched
    // cold, ~0.9 us per row (P0 finish at 24 rows 8.2 -> 2.8 us, the whole
    // call with L2 flushed 133 -> 120 us)
    float4 xs[RB][NACC], as[RB];
#pragma unroll
    for (int b = 0; b < RB; ++b) {
#pragma unroll
      for (int a = 0; a < NACC; ++a) {
        xs[b][a] = v[b][a][0];
#pragma unroll
        for (int sl = 1; sl < SMAX; ++sl) {  // slot order; the predicated-off slots add zero
          xs[b][a].x += v[b][a][sl].x;
          xs[b][a].y += v[b][a][sl].y;
          xs[b][a].z += v[b][a][sl].z;
          xs[b][a].w += v[b][a][sl].w;
        }
      }
      as[b] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (p == 2 && i0 + b < my_rows)
        as[b] = __ldcg(reinterpret_cast<const float4*>(L.hid + (int64_t)(w + 4 * (i0 + b)) * L.d + feat));
    }
#pragma unroll 1
    for (int b = 0; b < RB && i0 + b < my_rows; ++b) {  // the same in every lane of the warp
      const int32_t r = w + 4 * (i0 + b);
      if (NACC == 2)
        emit_gate(L, r, feat, xs[b][0], xs[b][NACC - 1], srow[r]);
      else if (p == 3)
        emit_argmax(L, r, feat, q, xs[b][0]);
      else
        emit_hidden(L, p, f, r, feat, q, xs[b][0], as[b], ga);
    }
  }
}

template <int NACC>
__device__ void finish_tile_n(const PredLaunch& L, int p, int32_t f, int32_t cnt, int et,
                              const float* srow) {
  switch (cnt) {  // the slot count fixes the batch shape (one batch for 24 rows up to 5 slots)
    case 1: finish_tile_t<1, NACC>(L, p, f, cnt, et, srow); break;
    case 2: finish_tile_t<2, NACC>(L, p, f, cnt, et, srow); break;
    case 3: finish_tile_t<3, NACC>(L, p, f, cnt, et, srow); break;
    case 4: finish_tile_t<4, NACC>(L, p, f, cnt, et, srow); break;
    case 5: finish_tile_t<5, NACC>(L, p, f, cnt, et, srow); break;
    case 6: finish_tile_t<6, NACC>(L, p, f, cnt, et, srow); break;
    default: finish_tile_t<8, NACC>(L, p, f, cnt, et, srow); break;
  }
}

__device__ void finish_tile_any(const PredLaunch& L, int p, int32_t f, int32_t cnt, int et,
                                const float* srow) {
  if (p == 1)
    finish_tile_n<2>(L, p, f, cnt, et, srow);
  else
    finish_tile_n<1>(L, p, f, cnt, et, srow);
}

// The row scales s(A) = 1 / sqrt(mean(A^2) + eps) of every row from the P0
// tiles' sums of squares, into srow (shared): four threads per row, each
// summing every fourth tile, then combined in a fixed order.
__device__ void row_scales(const PredLaunch& L, int et, float* srow) {
  const int k = et & 3;
  const int32_t nt = L.d / 128;
  for (int32_t r0 = 0; r0 < L.rows; r0 += kEpiThreads / 4) {
    const int32_t r = r0 + (et >> 2);
    float s = 0.f;
    if (r < L.rows)
#pragma unroll 8
      for (int32_t t = k; t < nt; t += 4) s += __ldcg(L.ss + (int64_t)t * 128 + r);
    s += __shfl_xor_sync(0xffffffffu, s, 1);
    s += __shfl_xor_sync(0xffffffffu, s, 2);
    if (r < L.rows && k == 0) srow[r] = 1.0f / sqrtf(s / (float)L.d + L.eps);
  }
}

// The epilogue warps' row scales: once every P0 tile is final (a bounded wait
// by one thread), s(A) of every row into srow.  False if the wait gave up or
// another role failed (every epilogue thread gets the same answer).
__device__ bool ensure_row_scales(const PredLaunch& L, int et, float* srow,
                                  volatile int32_t* fail) {
  bool stop = false;
  if (et == 0) {
    stop = *fail != 0 || !wait_count(L, done_ctr(L, 0), (uint32_t)L.ph[0].tiles + L.shortfall);
    if (stop) *fail = 1;
  }
  if (bar_or(kBarEpi, kEpiThreads, stop)) return false;
  fence_acq_rel_gpu();
  row_scales(L, et, srow);
  bar_named(kBarEpi, kEpiThreads);
  return true;
}

__device__ __forceinline__ void issue_weights(const PredLaunch& L, int p, int32_t u,
                                              unsigned char* dst, uint64_t* bar, uint64_t pol,
                                              const CUtensorMap* tmW0, const CUtensorMap* tmW1,
                                              const CUtensorMap* tmW3, const CUtensorMap* tmW2,
                                              const CUtensorMap* tmWH) {
  const PredPhase& ph = L.ph[p];
  const int32_t f = u / ph.upt, j = u - f * ph.upt;
  if (p == 0) {
    tma_load_3d(dst, tmW0, 0, f * 128, 2 * j, bar, pol);
  } else if (p == 1) {
    tma_load_2d(dst, tmW1, j * 64, f * 128, bar, pol);
    tma_load_2d(dst + 16384, tmW3, j * 64, f * 128, bar, pol);
  } else if (p == 2) {
    tma_load_3d(dst, tmW2, 0, f * 128, 2 * j, bar, pol);
  } else {
    tma_load_3d(dst, tmWH, 0, j * 128, 2 * f, bar, pol);
  }
}

// The activation tile of unit u: rows x kw entries of the phase's input from
// column j * kw, as [kw / 64][nn rows][128 B] (rows past `rows` read as zero).
__device__ __forceinline__ void issue_x(const PredLaunch& L, int p, int32_t u, unsigned char* dst,
                                        uint64_t* bar, uint64_t pol, const CUtensorMap* tmZ,
                                        const CUtensorMap* tmAg, const CUtensorMap* tmG,
                                        const CUtensorMap* tmHg) {
  const PredPhase& ph = L.ph[p];
  const int32_t j = u % ph.upt;
  if (p == 0)
    tma_load_3d(dst, tmZ, 0, 0, 2 * j, bar, pol);
  else if (p == 1)
    tma_load_2d(dst, tmAg, j * 64, 0, bar, pol);  // box {64, nn}
  else if (p == 2)
    tma_load_3d(dst, tmG, 0, 0, 2 * j, bar, pol);
  else
    tma_load_3d(dst, tmHg, 0, 0, 2 * j, bar, pol);  // the 3D view of the same array
}

}  // namespace

namespace {

__global__ void __launch_bounds__(kPThreads, 1)
predictor_kernel(const __grid_constant__ CUtensorMap tmW0, const __grid_constant__ CUtensorMap tmW1,
                 const __grid_constant__ CUtensorMap tmW3, const __grid_constant__ CUtensorMap tmW2,
                 const __grid_constant__ CUtensorMap tmWH, const __grid_constant__ CUtensorMap tmZ,
                 const __grid_constant__ CUtensorMap tmAg, const __grid_constant__ CUtensorMap tmG,
                 const __grid_constant__ CUtensorMap tmHg, PredLaunch L) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  // ring slot: the unit's weights (32 KB), then its activation tile (two
  // 64-wide K atoms of nn rows); one barrier per slot for both
  const int S = L.stages;
  const uint32_t xslot = (uint32_t)L.nn * 256u;
  const uint32_t slot_bytes = kUnitBytes + xslot;
  unsigned char* ring = smem;
  uint64_t* full = reinterpret_cast<uint64_t*>(ring + S * slot_bytes);
  uint64_t* empty = full + S;
  uint64_t* acc_full = empty + S;      // [2]
  uint64_t* acc_empty = acc_full + 2;  // [2]
  uint64_t* mma_done = acc_empty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_done + 1);
  // a role that gives up raises `fail`; the epilogue warps decide to stop only
  // through a reducing named barrier (bar_or), so they leave their loop together
  volatile int32_t* fail = reinterpret_cast<volatile int32_t*>(tmem_slot + 1);
  uint32_t* bcast = reinterpret_cast<uint32_t*>(tmem_slot + 2);  // [2]
  float* srow = reinterpret_cast<float*>(tmem_slot + 8);          // [128]

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int32_t cta = blockIdx.x;
  uint32_t ncols = 32;
  while (ncols < (uint32_t)(4 * L.nc)) ncols <<= 1;

  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 2);  // the weight producer's and the activation producer's arrivals
      mbar_init(&empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&acc_full[s], 1);
      mbar_init(&acc_empty[s], 4);  // one arrival per epilogue warp
    }
    mbar_init(mma_done, 1);
    *fail = 0;
    fence_barrier_init();
  }
  if (warp == kWarpMma && lane < 9) {  // the descriptors of the first copies of every phase
    const CUtensorMap* map = lane == 0 ? &tmW0 : lane == 1 ? &tmW1 : lane == 2 ? &tmW3
                           : lane == 3 ? &tmW2 : lane == 4 ? &tmWH : lane == 5 ? &tmZ
                           : lane == 6 ? &tmAg : lane == 7 ? &tmG : &tmHg;
    prefetch_tensormap(map);
  }
  if (warp == kWarpX) {
    tmem_alloc(tmem_slot, ncols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp <= 1) {
    // ---- weight producers: unit gu (counted over all phases) is issued by
    // warp gu % 2 into ring slot gu % S
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      uint32_t gu = 0;
      bool ok = true;
      for (int p = 0; p < kPhases && ok; ++p) {
        const PredPhase& ph = L.ph[p];
        const int64_t lo = unit_start(cta, ph.units, L.ncta), hi = unit_start(cta + 1, ph.units, L.ncta);
        for (int64_t u = lo; u < hi; ++u, ++gu) {
          if ((int)(gu & 1u) != warp) continue;
          const uint32_t s = gu % S;
          if (*fail || (gu >= (uint32_t)S &&
                        !mbar_wait(&empty[s], ((gu / S) - 1) & 1, L.status, L.max_polls))) {
            *fail = 1;
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&full[s], kUnitBytes);
          issue_weights(L, p, (int32_t)u, ring + s * slot_bytes, &full[s], pol, &tmW0, &tmW1,
                        &tmW3, &tmW2, &tmWH);
        }
      }
      // copies still in flight can only be among the last S units issued:
      // wait for those before the CTA may exit
      for (uint32_t x = gu > (uint32_t)S ? gu - S : 0; x < gu; ++x)
        if ((int)(x & 1u) == warp) mbar_wait(&full[x % S], (x / S) & 1, nullptr, L.max_polls);
    }
    __syncwarp();
  } else if (warp == kWarpX) {
    // ---- activation producer: lane 0 issues the copies.  Per-tile waits:
    // to learn which tiles of the previous phase are final, every lane polls
    // one tile of a window of 32 starting at the one the next unit reads, so
    // one round trip answers for the units that follow.
    const uint64_t pol = policy_evict_last();  // read again by the CTAs sharing a K range
    uint32_t gu = 0;
    bool ok = true;
    for (int p = 0; p < kPhases && ok; ++p) {
      const PredPhase& ph = L.ph[p];
      int32_t wbase = -1;  // tiles wbase + k of the previous phase are final for the bits k of wmask
      uint32_t wmask = 0;
      bool all_final = p == 0;  // P0 reads z
      if (p >= 1 && !L.tile_waits) {  // every tile of the previous phase final first
        bool got = true;
        if (lane == 0) {
          got = *fail == 0 &&
                wait_count(L, done_ctr(L, p - 1), (uint32_t)L.ph[p - 1].tiles + L.shortfall);
          if (!got) *fail = 1;
          fence_proxy_async_global();
        }
        if (!__shfl_sync(0xffffffffu, got, 0)) {
          ok = false;
          break;
        }
        all_final = true;
      }
      const uint32_t bytes = (uint32_t)L.nn * ph.kw * 2;
      const int64_t lo = unit_start(cta, ph.units, L.ncta), hi = unit_start(cta + 1, ph.units, L.ncta);
      for (int64_t u = lo; u < hi; ++u, ++gu) {
        const uint32_t s = gu % S;
        if (!all_final) {
          const int32_t need = (int32_t)((u % ph.upt) * ph.kw / 128);
          if (!(need >= wbase && need < wbase + 32 && ((wmask >> (need - wbase)) & 1u))) {
            const PredPhase& pp = L.ph[p - 1];
            const int32_t t = need + lane;
            uint32_t target = 0xffffffffu;  // a tile past the end is never final
            if (t < pp.tiles) {
              const int32_t c0 = unit_cta((int64_t)t * pp.upt, pp.units, L.ncta);
              const int32_t c1 = unit_cta((int64_t)(t + 1) * pp.upt - 1, pp.units, L.ncta);
              target = (uint32_t)(c1 - c0 + 2) + L.shortfall;  // every contributor, then the finisher
            }
            wbase = need;
            wmask = 0;
            bool got = false, stop = *fail != 0;
            for (uint32_t i = 0; i < L.max_polls && !stop; ++i) {
              const bool f = target != 0xffffffffu && !((wmask >> lane) & 1u) &&
                             ld_acquire_u32(ticket(L, p - 1, t)) >= target;
              wmask |= __ballot_sync(0xffffffffu, f);
              if (wmask & 1u) {
                got = true;
                break;
              }
              if ((i & 1023u) == 1023u)
                stop = __shfl_sync(0xffffffffu, lane == 0 && ld_acquire_u32(abort_flag(L)) != 0u, 0);
              if (i > 64) __nanosleep(128);
            }
            __syncwarp();
            if (lane == 0) {
              if (got) {
                got = ld_acquire_u32(abort_flag(L)) == 0u;
              } else if (!stop) {  // the poll limit ran out
                atomicExch(abort_flag(L), 1u);
                record_status(L.status, SSD_ERR_TIMEOUT);
              }
              if (!got) *fail = 1;
              // the acquiring lanes' loads before the copies of this lane
              fence_acq_rel_gpu();
              fence_proxy_async_global();
            }
            if (!__shfl_sync(0xffffffffu, got, 0)) {
              ok = false;
              break;
            }
          }
        }
        if (lane == 0) {
          if (*fail || (gu >= (uint32_t)S &&
                        !mbar_wait(&empty[s], ((gu / S) - 1) & 1, L.status, L.max_polls))) {
            *fail = 1;
            ok = false;
          } else {
            mbar_arrive_expect_tx(&full[s], bytes);
            issue_x(L, p, (int32_t)u, ring + s * slot_bytes + kUnitBytes, &full[s], pol, &tmZ,
                    &tmAg, &tmG, &tmHg);
          }
        }
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) break;
      }
    }
    if (lane == 0)
      for (uint32_t x = gu > (uint32_t)S ? gu - S : 0; x < gu; ++x)
        mbar_wait(&full[x % S], (x / S) & 1, nullptr, L.max_polls);
    __syncwarp();
  } else if (warp == kWarpMma) {
    // ---- MMA issue: one thread
    if (lane == 0) {
      const uint32_t idk = idesc_bf16(128, L.nn, false, false);
      const uint32_t idmn = idesc_bf16(128, L.nn, true, false);
      const uint32_t xatom = (uint32_t)L.nn * 128u;  // one 64-wide K atom of the activations
      uint32_t gu = 0, tc = 0;
      bool ok = true;
      for (int p = 0; p < kPhases && ok; ++p) {
        const PredPhase& ph = L.ph[p];
        const int64_t lo = unit_start(cta, ph.units, L.ncta), hi = unit_start(cta + 1, ph.units, L.ncta);
        uint32_t buf = 0;
        int32_t j = (int32_t)(lo % ph.upt);  // K step of unit u inside its tile
        for (int64_t u = lo; u < hi; ++u, ++gu, j = (j + 1 == ph.upt) ? 0 : j + 1) {
          const bool first = (u == lo) || j == 0;
          const bool last = (u == hi - 1) || j == ph.upt - 1;
          if (first) {
            buf = tc & 1u;
            if (tc >= 2 && !mbar_wait(&acc_empty[buf], ((tc >> 1) - 1) & 1, L.status, L.max_polls)) {
              ok = false;
              break;
            }
          }
          if (!mbar_wait(&full[gu % S], (gu / S) & 1, L.status, L.max_polls)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t wb = smem_u32(ring + (gu % S) * slot_bytes);
          const uint64_t dx = smem_desc(wb + kUnitBytes, 16, 1024);
          const uint32_t dacc = tmem + buf * 2u * (uint32_t)L.nc;
          const uint32_t a0 = first ? 0u : 1u;
          if (p == 1) {  // W1 and W3 tiles of 64 K against one activation atom
            const uint64_t dw = smem_desc(wb, 16, 1024);
#pragma unroll
            for (int kk = 0; kk < 4; ++kk) {
              const uint32_t acc = kk > 0 ? 1u : a0;
              mma_ss(dacc, smem_desc_at(dw, kk * 32), smem_desc_at(dx, kk * 32), idk, acc);
              mma_ss(dacc + L.nc, smem_desc_at(dw, 16384 + kk * 32), smem_desc_at(dx, kk * 32), idk,
                     acc);
            }
          } else if (p == 3) {  // GenHead: vocabulary contiguous (MN-major), halves 16 KB apart
            const uint64_t dw = smem_desc(wb, 16384, 1024);
#pragma unroll
            for (int kk = 0; kk < 8; ++kk)
              mma_ss(dacc, smem_desc_at(dw, kk * 2048),
                     smem_desc_at(dx, (kk >> 2) * xatom + (kk & 3) * 32), idmn, kk > 0 ? 1u : a0);
          } else {  // K-major: two 64-wide K atoms of 16 KB
            const uint64_t dw = smem_desc(wb, 16, 1024);
#pragma unroll
            for (int kk = 0; kk < 8; ++kk)
              mma_ss(dacc, smem_desc_at(dw, (kk >> 2) * 16384 + (kk & 3) * 32),
                     smem_desc_at(dx, (kk >> 2) * xatom + (kk & 3) * 32), idk, kk > 0 ? 1u : a0);
          }
          mma_commit(&empty[gu % S]);
          if (last) {
            mma_commit(&acc_full[buf]);
            ++tc;
          }
        }
      }
      if (!ok) *fail = 1;
      mma_commit(mma_done);  // arrives once every MMA issued above has completed
    }
    __syncwarp();
  } else {
    // ---- epilogue (warps 4-7): TMEM lane = feature et of the tile
    const int et = tid - kEpiWarp0 * 32;
    const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
    uint32_t tc = 0;
    bool ok = true, have_scales = false;
    for (int p = 0; p < kPhases && ok; ++p) {
      const PredPhase& ph = L.ph[p];
      const int nacc = p == 1 ? 2 : 1;
      if (p == 1 && !L.tile_waits) {
        // per-phase waits: the P1 products start once every P0 tile is final,
        // so the row scales are summed then, beside the first products
        if (!ensure_row_scales(L, et, srow, fail)) {
          ok = false;
          break;
        }
        have_scales = true;
      }
      const int64_t lo = unit_start(cta, ph.units, L.ncta), hi = unit_start(cta + 1, ph.units, L.ncta);
      const int32_t f0 = (int32_t)(lo / ph.upt), f1 = (int32_t)((hi - 1) / ph.upt);
      for (int32_t f = f0; f <= f1; ++f, ++tc) {
        const uint32_t buf = tc & 1u;
        bool stop = false;
        if (lane == 0) {
          stop = *fail != 0 || !mbar_wait(&acc_full[buf], (tc >> 1) & 1, L.status, L.max_polls);
          if (stop) *fail = 1;
        }
        if (bar_or(kBarEpi, kEpiThreads, stop)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const int32_t first = unit_cta((int64_t)f * ph.upt, ph.units, L.ncta);
        const int32_t lastc = unit_cta((int64_t)(f + 1) * ph.upt - 1, ph.units, L.ncta);
        float* dst = L.part + (p & 1) * L.part_odd +
                     ((int64_t)f * ph.slots + (cta - first)) * nacc * L.nn * 128 + et;
        for (int a = 0; a < nacc; ++a) {
          for (int32_t ch = 0; ch < L.nc / 32; ++ch) {
            float v[32];
            tmem_ld32(tmem + lane_base + buf * 2u * (uint32_t)L.nc + a * L.nc + ch * 32, v);
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const int32_t r = ch * 32 + i;
              if (r < L.rows) __stcg(dst + ((int64_t)a * L.nn + r) * 128, v[i]);
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&acc_empty[buf]);
        fence_acq_rel_gpu();  // the partial before the ticket
        bar_named(kBarEpi, kEpiThreads);
        if (et == 0) bcast[0] = atomicAdd(ticket(L, p, f), 1u);
        bar_named(kBarEpi, kEpiThreads);
        if (bcast[0] != (uint32_t)(lastc - first)) continue;  // not the last contributor
        fence_acq_rel_gpu();  // every contributor's partial after the ticket
        if (p == 1 && !have_scales) {  // per-tile waits: before the CTA's first P1 finish
          if (!ensure_row_scales(L, et, srow, fail)) {
            ok = false;
            break;
          }
          have_scales = true;
        }
        finish_tile_any(L, p, f, lastc - first + 1, et, srow);
        fence_proxy_async_global();  // Ag, G, Hg are loaded by TMA in the next phase
        fence_acq_rel_gpu();
        bar_named(kBarEpi, kEpiThreads);
        if (et == 0) {
          // the tile is final (a reduction: nothing waits for its result)
          asm volatile("red.relaxed.gpu.global.add.u32 [%0], 1;" ::"l"(ticket(L, p, f)) : "memory");
          bcast[1] = atomicAdd(done_ctr(L, p), 1u);
        }
        bar_named(kBarEpi, kEpiThreads);
        if (p == 3 && bcast[1] == (uint32_t)(ph.tiles - 1)) {
          // the last tile of the vocabulary: every tile's key is in
          fence_acq_rel_gpu();
          for (int32_t r = et; r < L.rows; r += kEpiThreads) L.out_tok[r] = argmax_index(__ldcg(L.best + (int64_t)r * kKeyStride));
        }
      }
    }
  }

  // ---- teardown: every MMA complete before tensor memory is freed
  if (warp == kWarpX && lane == 0) mbar_wait(mma_done, 0, nullptr, L.max_polls);
  tc_fence_before();
  __syncthreads();
  if (warp == kWarpX) {
    tc_fence_after();
    tmem_dealloc(tmem, ncols);
  }
}

}  // namespace

namespace {

size_t al256(size_t x) { return (x + 255) & ~size_t(255); }

struct PredPlan {
  PredPhase ph[kPhases];
  int32_t ncta, nn, nc, stages, max_tiles;
  size_t part_floats, part_odd, smem;
};

int32_t tile_slots(const PredPhase& ph, int32_t ncta) {
  int32_t most = 1;
  for (int32_t f = 0; f < ph.tiles; ++f) {
    const int64_t u0 = (int64_t)f * ph.upt, u1 = (int64_t)(f + 1) * ph.upt - 1;
    const int32_t c0 = (int32_t)(((u0 + 1) * ncta + ph.units - 1) / ph.units) - 1;
    const int32_t c1 = (int32_t)(((u1 + 1) * ncta + ph.units - 1) / ph.units) - 1;
    most = std::max(most, c1 - c0 + 1);
  }
  return most;
}

PredPlan make_plan(int32_t rows, int32_t d, int32_t m, int32_t V, int32_t sm_count) {
  PredPlan P;
  // P0: W0 [d][2d]; P1: W1, W3 [m][d] in 64-wide K steps; P2: W2 [d][m];
  // P3: W_head [d][V] (vocabulary on M)
  const int32_t tiles[kPhases] = {d / 128, m / 128, d / 128, V / 128};
  const int32_t K[kPhases] = {2 * d, d, m, d};
  const int32_t kw[kPhases] = {128, 64, 128, 128};
  int32_t min_units = INT32_MAX;
  for (int p = 0; p < kPhases; ++p) {
    P.ph[p].tiles = tiles[p];
    P.ph[p].kw = kw[p];
    P.ph[p].upt = K[p] / kw[p];
    P.ph[p].units = tiles[p] * P.ph[p].upt;
    min_units = std::min(min_units, P.ph[p].units);
  }
  // every CTA takes at least one unit of every phase, and no tile is split over
  // more than kMaxSlots CTAs (the finisher sums at most that many partials)
  P.ncta = std::max(1, std::min(sm_count, min_units));
  if (rows > kTileWaitRows) {
    // many rows: the tiles' finishes, not the stream, set the phase
    // boundaries, so take the largest CTA count (down to 3/4 of the SMs) that
    // divides every phase's units: every CTA's range then starts and ends on
    // a tile boundary, so a tile's contributors end together and fewer of them
    // share it (at the paper's sizes 128 CTAs: 4, 2, 4 and 1 per tile)
    for (int32_t c = P.ncta; c >= (P.ncta * 3) / 4 && c >= 1; --c) {
      bool all = true;
      for (int p = 0; p < kPhases; ++p) all = all && (P.ph[p].units % c == 0);
      if (all) {
        P.ncta = c;
        break;
      }
    }
  }
  for (;;) {
    int32_t most = 1;
    for (int p = 0; p < kPhases; ++p) most = std::max(most, tile_slots(P.ph[p], P.ncta));
    if (most <= kMaxSlots || P.ncta == 1) break;
    --P.ncta;
  }
  P.max_tiles = 0;
  size_t part_max[2] = {0, 0};
  P.nn = (rows + 15) / 16 * 16;
  P.nc = (P.nn + 31) / 32 * 32;
  for (int p = 0; p < kPhases; ++p) {
    P.ph[p].slots = tile_slots(P.ph[p], P.ncta);
    P.max_tiles = std::max(P.max_tiles, P.ph[p].tiles);
    const size_t nacc = p == 1 ? 2 : 1;
    part_max[p & 1] = std::max(part_max[p & 1],
                               (size_t)P.ph[p].tiles * P.ph[p].slots * nacc * P.nn * 128);
  }
  P.part_odd = (part_max[0] + 63) / 64 * 64;
  P.part_floats = P.part_odd + part_max[1];
  const size_t slot = (size_t)kUnitBytes + (size_t)P.nn * 256;
  const size_t budget = 232448;  // 227 KB of dynamic shared memory per CTA
  P.stages = (int32_t)std::min<size_t>(8, (budget - 1024 - 2048) / slot);
  P.smem = 1024 + (size_t)P.stages * slot + (2 * P.stages + 5) * 8 + 32 + kMaxRows * 4;
  return P;
}

struct PredWs {
  unsigned int* ctr;
  unsigned long long* best;  // after the counters: zeroed with them
  size_t zero_bytes;         // counters and keys
  float* part;
  float* ss;
  __nv_bfloat16* ag;
  __nv_bfloat16* g;
  float* hid;
  size_t bytes;
};

PredWs carve(const PredPlan& P, int32_t rows, int32_t d, int32_t m, int32_t V, bool own_hidden,
             void* base) {
  PredWs w;
  unsigned char* b = static_cast<unsigned char*>(base);
  size_t off = 0;
  auto take = [&](size_t n) {
    unsigned char* p = b + off;
    off += al256(n);
    return p;
  };
  const size_t ctr_bytes = al256((size_t)(kPhases * P.max_tiles + kPhases + 1) * kCtrStride * 4);
  w.zero_bytes = ctr_bytes + (size_t)kMaxRows * kKeyStride * 8;
  w.ctr = reinterpret_cast<unsigned int*>(take(w.zero_bytes));
  w.best = reinterpret_cast<unsigned long long*>(reinterpret_cast<unsigned char*>(w.ctr) + ctr_bytes);
  w.part = reinterpret_cast<float*>(take(P.part_floats * 4));
  w.ss = reinterpret_cast<float*>(take((size_t)(d / 128) * 128 * 4));
  w.ag = reinterpret_cast<__nv_bfloat16*>(take((size_t)rows * d * 2));
  w.g = reinterpret_cast<__nv_bfloat16*>(take((size_t)rows * m * 2));
  w.hid = own_hidden ? reinterpret_cast<float*>(take((size_t)rows * d * 4)) : nullptr;
  w.bytes = off;
  return w;
}

bool shapes_ok(int32_t rows, int32_t d, int32_t m, int32_t V) {
  return rows >= 1 && rows <= kMaxRows && d >= 128 && m >= 128 && V >= 128 && d % 128 == 0 &&
         m % 128 == 0 && V % 128 == 0;
}

// One launch over at most kMaxRows rows.
cudaError_t launch_rows(const PredictorArgs& a, void* ws, size_t ws_bytes, int32_t* status,
                        cudaStream_t stream) {
  if (!shapes_ok(a.rows, a.d, a.m, a.V)) return cudaErrorInvalidValue;
  const PredPlan P = make_plan(a.rows, a.d, a.m, a.V, device_sm_count());
  const PredWs w = carve(P, a.rows, a.d, a.m, a.V, a.out_hidden == nullptr, ws);
  if (ws == nullptr || ws_bytes < w.bytes) return cudaErrorInvalidValue;

  PredLaunch L;
  for (int p = 0; p < kPhases; ++p) L.ph[p] = P.ph[p];
  L.ncta = P.ncta;
  L.rows = a.rows;
  L.nn = P.nn;
  L.nc = P.nc;
  L.stages = P.stages;
  L.d = a.d;
  L.m = a.m;
  L.V = a.V;
  L.max_polls = wait_poll_limit();
  L.shortfall = barrier_shortfall();
  // measured (graphs of back-to-back calls): per-tile waits 136 vs 144 us at 72
  // rows, 147 vs 145 at 90, 150 vs 148 at 128
  L.tile_waits = a.rows <= kTileWaitRows;
  L.eps = a.eps;
  L.gamma1 = a.gamma1;
  L.gamma2 = a.gamma2;
  L.hid = a.out_hidden != nullptr ? a.out_hidden : w.hid;
  L.ag = w.ag;
  L.g = w.g;
  L.ss = w.ss;
  L.best = w.best;
  L.part = w.part;
  L.part_odd = (int64_t)P.part_odd;
  L.ctr = w.ctr;
  L.max_tiles = P.max_tiles;
  L.out_tok = a.out_tok;
  L.status = status;

  const uint64_t d = (uint64_t)a.d, m = (uint64_t)a.m, V = (uint64_t)a.V, R = (uint64_t)a.rows;
  const uint32_t nn = (uint32_t)P.nn;
  CUtensorMap t0, t1, t3, t2, th, tz, tag, tg, thg;
  bool ok = true;
  {  // W0 [d][2d]: {64, d rows, 2d / 64 column blocks}, box {64, 128, 2}
    const uint64_t dims[3] = {64, d, 2 * d / 64}, str[2] = {2 * d * 2, 128};
    const uint32_t box[3] = {64, 128, 2};
    ok = ok && bf16_tensor_map(&t0, a.w0, 3, dims, str, box);
  }
  {  // W1, W3 [m][d]: {d, m}, box {64, 128}
    const uint64_t dims[2] = {d, m}, str[1] = {d * 2};
    const uint32_t box[2] = {64, 128};
    ok = ok && bf16_tensor_map(&t1, a.w1, 2, dims, str, box) &&
         bf16_tensor_map(&t3, a.w3, 2, dims, str, box);
  }
  {  // W2 [d][m]: {64, d rows, m / 64}, box {64, 128, 2}
    const uint64_t dims[3] = {64, d, m / 64}, str[2] = {m * 2, 128};
    const uint32_t box[3] = {64, 128, 2};
    ok = ok && bf16_tensor_map(&t2, a.w2, 3, dims, str, box);
  }
  {  // W_head [d][V]: {64 vocabulary entries, d rows, V / 64}, box {64, 128 K, 2}
    const uint64_t dims[3] = {64, d, V / 64}, str[2] = {V * 2, 128};
    const uint32_t box[3] = {64, 128, 2};
    ok = ok && bf16_tensor_map(&th, a.w_head, 3, dims, str, box);
  }
  {  // activations [rows][K] as {64, rows, K / 64}, box {64, nn, 2}: [2][nn][128 B]
    const uint32_t box[3] = {64, nn, 2};
    const uint64_t dz[3] = {64, R, 2 * d / 64}, sz[2] = {2 * d * 2, 128};
    const uint64_t dg[3] = {64, R, m / 64}, sg[2] = {m * 2, 128};
    const uint64_t dh[3] = {64, R, d / 64}, sh[2] = {d * 2, 128};
    ok = ok && bf16_tensor_map(&tz, a.z, 3, dz, sz, box) &&
         bf16_tensor_map(&tg, w.g, 3, dg, sg, box) && bf16_tensor_map(&thg, w.ag, 3, dh, sh, box);
    // Ag in 64-wide K steps (P1): {d, rows}, box {64, nn}
    const uint64_t da[2] = {d, R}, sa[1] = {d * 2};
    const uint32_t ba[2] = {64, nn};
    ok = ok && bf16_tensor_map(&tag, w.ag, 2, da, sa, ba);
  }
  if (!ok) return cudaErrorInvalidValue;
  cudaError_t e = cudaMemsetAsync(w.ctr, 0, w.zero_bytes, stream);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(predictor_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)P.smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)P.ncta, 1, 1);
  cfg.blockDim = dim3(kPThreads, 1, 1);
  cfg.dynamicSmemBytes = P.smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, predictor_kernel, t0, t1, t3, t2, th, tz, tag, tg, thg, L);
}

}  // namespace

size_t predictor_workspace(int32_t rows, int32_t d, int32_t m, int32_t V, bool own_hidden) {
  // more rows run as several launches over one workspace: launches of
  // kMaxRows rows and a last one of the rest, whose plan may differ
  const int32_t full = std::min(rows, kMaxRows), rest = rows > kMaxRows ? rows % kMaxRows : 0;
  if (!shapes_ok(full, d, m, V)) return 0;
  const int sm = device_sm_count();
  size_t bytes = carve(make_plan(full, d, m, V, sm), full, d, m, V, own_hidden, nullptr).bytes;
  if (rest > 0)
    bytes = std::max(bytes,
                     carve(make_plan(rest, d, m, V, sm), rest, d, m, V, own_hidden, nullptr).bytes);
  return bytes;
}

bool predictor_supported(int32_t d, int32_t m, int32_t V) { return shapes_ok(1, d, m, V); }

cudaError_t launch_predictor(const PredictorArgs& a, void* ws, size_t ws_bytes, int32_t* status,
                             cudaStream_t stream) {
  for (int32_t r0 = 0; r0 < a.rows; r0 += kMaxRows) {
    PredictorArgs c = a;
    c.rows = std::min(kMaxRows, a.rows - r0);
    c.z = static_cast<const __nv_bfloat16*>(a.z) + (int64_t)r0 * 2 * a.d;
    c.out_tok = a.out_tok + r0;
    c.out_hidden = a.out_hidden != nullptr ? a.out_hidden + (int64_t)r0 * a.d : nullptr;
    const cudaError_t e = launch_rows(c, ws, ws_bytes, status, stream);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace ssd
