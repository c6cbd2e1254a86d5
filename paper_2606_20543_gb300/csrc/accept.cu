// accept.cu — vocabulary-wide acceptance (steps a3-a5): target/draft softmax,
// the ratio at the draft token, the accept decision and, on rejection, the
// residual draw (Sec. 3.3 "Verification as Auto Correction", strategy (C)):
//   accept t with probability min(p(t) / q(t), 1); otherwise draw from
//   [p - q]_+ / sum [p - q]_+ (inverse CDF in vocabulary order, one uniform).
//
// Design (GB300): one CTA of 256 threads per row, no shared-memory copy of
// the row (so many rows stream at once).  Pass A reads both logit rows from
// HBM once with 16-byte loads, four per row per thread in flight, and keeps
// online (max, sum of 2^x) statistics and the first argmax in registers; one
// block reduction in a fixed order gives the log-sum-exps and the draft
// token, and thread 0 takes the decision.  Only rejected rows run pass B: the
// rows are re-read from L2 (they were read microseconds earlier; these loads
// mark the lines evict-first), the residual weights are formed with MUFU
// exp2, and the mass of every 128-entry chunk goes to shared memory in
// vocabulary order.  Warp 0 scans the chunk masses, finds the chunk holding
// u_res * Z, and re-walks that chunk to pick the token.
#include "kernels.cuh"

namespace ssd {

namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kUnroll = 4;             // float4 loads per row per thread in flight
constexpr int kMaxV = 1 << 20;         // chunk-mass table: V / 128 floats of shared memory
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// 2^x on the MUFU unit (results below 2^-126 flush to zero).
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Streaming 16-byte loads: the first read of a row keeps it in L2 for the
// residual pass; the residual pass marks its lines evict-first (last use).
__device__ __forceinline__ float4 ld_keep(const float4* p) {
  float4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.f32 {%0,%1,%2,%3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "l"(p));
  return v;
}
__device__ __forceinline__ float4 ld_last(const float4* p, uint64_t pol) {
  float4 v;
  asm volatile("ld.global.nc.L1::no_allocate.L2::cache_hint.v4.f32 {%0,%1,%2,%3}, [%4], %5;"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "l"(p), "l"(pol));
  return v;
}

__device__ __forceinline__ bool better_arg(float v, int32_t i, float bv, int32_t bi) {
  return v > bv || (v == bv && (uint32_t)i < (uint32_t)bi);
}

// Online (max, sum of exp2((x - max) * c)) over 4 more entries.
__device__ __forceinline__ void online4(float& m, float& s, const float4& x, float c) {
  const float mx = fmaxf(fmaxf(x.x, x.y), fmaxf(x.z, x.w));
  if (mx > m) {
    s *= ex2((m - mx) * c);  // m == -inf: s is 0 and stays 0
    m = mx;
  }
  if (m != -INFINITY) {
    const float mc = m * c;
    s += (ex2(fmaf(x.x, c, -mc)) + ex2(fmaf(x.y, c, -mc))) +
         (ex2(fmaf(x.z, c, -mc)) + ex2(fmaf(x.w, c, -mc)));
  }
}

// Merge two (max, sum) pairs.
__device__ __forceinline__ void merge(float& m, float& s, float m2, float s2, float c) {
  const float mn = fmaxf(m, m2);
  if (mn == -INFINITY) return;
  s = s * ex2((m - mn) * c) + s2 * ex2((m2 - mn) * c);
  m = mn;
}

// Residual weights of 4 entries: [p - q]_+ with p = 2^(x_p c - Cp), q = 2^(x_q c - Cq),
// or p itself for the draw from p.
__device__ __forceinline__ float4 weights4(const float4& xp, const float4& xq, float c, float Cp,
                                           float Cq, bool from_p) {
  float4 w;
  if (from_p) {
    w.x = ex2(fmaf(xp.x, c, -Cp));
    w.y = ex2(fmaf(xp.y, c, -Cp));
    w.z = ex2(fmaf(xp.z, c, -Cp));
    w.w = ex2(fmaf(xp.w, c, -Cp));
  } else {
    w.x = fmaxf(ex2(fmaf(xp.x, c, -Cp)) - ex2(fmaf(xq.x, c, -Cq)), 0.f);
    w.y = fmaxf(ex2(fmaf(xp.y, c, -Cp)) - ex2(fmaf(xq.y, c, -Cq)), 0.f);
    w.z = fmaxf(ex2(fmaf(xp.z, c, -Cp)) - ex2(fmaf(xq.z, c, -Cq)), 0.f);
    w.w = fmaxf(ex2(fmaf(xp.w, c, -Cp)) - ex2(fmaf(xq.w, c, -Cq)), 0.f);
  }
  return w;
}

struct Shared {
  float red[kWarps][4];
  int32_t red_i[kWarps];
  float Cp, Cq;      // log2-domain normalisers: max * c + log2(sum)
  int32_t accept;    // 1 accepted, 0 rejected, 2 no valid draft token
  float u_res;
};

// One CTA per row.  Pass A streams both logit rows once from HBM and keeps
// online statistics; pass B (rejected rows only) re-reads them from L2,
// computes the residual weights and the mass of every 128-entry chunk (warp w
// of iteration k owns entries [(8k + w) * 128, +128), so chunks are in
// vocabulary order); warp 0 then scans the chunk masses and re-walks the
// chunk holding the CDF crossing.
__global__ void __launch_bounds__(kThreads, 4) accept_kernel(AcceptArgs a) {
  extern __shared__ float chunk_mass[];  // [V / 128] (rounded up to whole iterations)
  __shared__ Shared sh;
  const int32_t tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t r = blockIdx.x;

  // ---- rows outside the frontier (padding slots of a verification step)
  if (a.n_drafts != nullptr) {
    const int32_t b = (int32_t)(r / a.D_max), j = (int32_t)(r % a.D_max);
    if (j >= a.n_drafts[b]) {
      if (tid == 0) {
        a.out_tok[r] = -1;
        a.accepted[r] = 0;
        if (a.ratio) a.ratio[r] = 0.f;
        if (a.lse) { a.lse[2 * r] = 0.f; a.lse[2 * r + 1] = 0.f; }
      }
      return;
    }
  }
  int32_t given_t = -1;
  if (a.draft_tok != nullptr) {
    given_t = a.draft_tok[r];
    if (given_t < 0 || given_t >= a.V) {
      if (tid == 0) {
        record_status(a.status, SSD_ERR_DEVICE_BOUNDS);
        a.out_tok[r] = -1;
        a.accepted[r] = 0;
        if (a.ratio) a.ratio[r] = 0.f;
      }
      return;
    }
  }

  const float4* tp = reinterpret_cast<const float4*>(a.tgt + r * a.ld);
  const float4* dp = reinterpret_cast<const float4*>(a.drf + r * a.ld);
  const int32_t nv = a.V >> 2;
  const float c = kLog2e / a.temperature;

  // ---- pass A: online max / sum-exp of both rows, first argmax of the draft row
  float mp = -INFINITY, sp = 0.f, mq = -INFINITY, sq = 0.f;
  int32_t iq = 0x7fffffff;
  for (int32_t base = tid; base < nv; base += kThreads * kUnroll) {
    float4 xp[kUnroll], xq[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int32_t i = base + u * kThreads;
      if (i < nv) {
        xp[u] = ld_keep(tp + i);
        xq[u] = ld_keep(dp + i);
      } else {
        xp[u] = xq[u] = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
      }
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      online4(mp, sp, xp[u], c);
      // draft row: entries visited in ascending order, strict '>' keeps the first max
      const float4 x = xq[u];
      const float mx = fmaxf(fmaxf(x.x, x.y), fmaxf(x.z, x.w));
      if (mx > mq) {
        const int32_t e = 4 * (base + u * kThreads);
        iq = e + (x.x == mx ? 0 : x.y == mx ? 1 : x.z == mx ? 2 : 3);
      }
      online4(mq, sq, x, c);
    }
  }
  // block reduction (fixed order: xor tree in warps, then warps 0..7)
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    merge(mp, sp, __shfl_xor_sync(0xffffffffu, mp, o), __shfl_xor_sync(0xffffffffu, sp, o), c);
    const float om = __shfl_xor_sync(0xffffffffu, mq, o);
    const float os = __shfl_xor_sync(0xffffffffu, sq, o);
    const int32_t oi = __shfl_xor_sync(0xffffffffu, iq, o);
    const bool take = better_arg(om, oi, mq, iq);
    merge(mq, sq, om, os, c);
    if (take) iq = oi;
  }
  if (lane == 0) {
    sh.red[warp][0] = mp;
    sh.red[warp][1] = sp;
    sh.red[warp][2] = mq;
    sh.red[warp][3] = sq;
    sh.red_i[warp] = iq;
  }
  __syncthreads();
  if (tid == 0) {
    float Mp = sh.red[0][0], Sp = sh.red[0][1], Mq = sh.red[0][2], Sq = sh.red[0][3];
    int32_t t = sh.red_i[0];
    for (int w = 1; w < kWarps; ++w) {
      merge(Mp, Sp, sh.red[w][0], sh.red[w][1], c);
      const bool take = better_arg(sh.red[w][2], sh.red_i[w], Mq, t);
      merge(Mq, Sq, sh.red[w][2], sh.red[w][3], c);
      if (take) t = sh.red_i[w];
    }
    if (given_t >= 0) t = given_t;
    const bool valid_t = t >= 0 && t < a.V;
    float ratio = 0.f;
    bool acc = false;
    const float2 u = row_uniforms(a.rng, r);
    if (valid_t) {
      const float xp_t = a.tgt[r * a.ld + t];  // L2-resident after pass A
      const float xq_t = a.drf[r * a.ld + t];
      const float l2p = (xp_t - Mp) * c - log2f(Sp);
      const float l2q = (xq_t - Mq) * c - log2f(Sq);
      ratio = exp2f(l2p - l2q);
      acc = u.x < fminf(ratio, 1.0f);
    } else {
      record_status(a.status, SSD_ERR_DEVICE_BOUNDS);  // non-finite logits
    }
    sh.accept = acc ? 1 : (valid_t ? 0 : 2);
    sh.u_res = u.y;
    sh.Cp = Mp * c + log2f(Sp);
    sh.Cq = Mq * c + log2f(Sq);
    a.accepted[r] = acc ? 1 : 0;
    if (acc) a.out_tok[r] = t;
    else if (!valid_t) a.out_tok[r] = -1;
    if (a.ratio) a.ratio[r] = ratio;
    if (a.lse) {
      a.lse[2 * r] = Mp / a.temperature + log2f(Sp) * kLn2;
      a.lse[2 * r + 1] = Mq / a.temperature + log2f(Sq) * kLn2;
    }
  }
  __syncthreads();
  if (sh.accept != 0) return;

  // ---- pass B: residual draw from [p - q]_+ (or from p when that mass is zero)
  const float Cp = sh.Cp, Cq = sh.Cq;
  const uint64_t pol = policy_evict_first();
  const int32_t iters = (nv + kThreads - 1) / kThreads;  // 1024 entries per iteration
  const int32_t nchunks = iters * kWarps;
  for (int pass = 0; pass < 2; ++pass) {
    const bool from_p = (pass == 1);
    for (int32_t k0 = 0; k0 < iters; k0 += kUnroll) {
      float4 xp[kUnroll], xq[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int32_t i = (k0 + u) * kThreads + tid;
        if (k0 + u < iters && i < nv) {
          xp[u] = ld_last(tp + i, pol);
          xq[u] = from_p ? xp[u] : ld_last(dp + i, pol);
        } else {
          xp[u] = xq[u] = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
        }
      }
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        if (k0 + u < iters) {
          const float4 w = weights4(xp[u], xq[u], c, Cp, Cq, from_p);
          const float m = warp_sum((w.x + w.y) + (w.z + w.w));
          if (lane == 0) chunk_mass[(k0 + u) * kWarps + warp] = m;
        }
      }
    }
    __syncthreads();
    if (warp == 0) {
      // chunk masses in vocabulary order: lane l owns chunks [l*per, (l+1)*per)
      const int32_t per = (nchunks + 31) / 32;
      float ls = 0.f;
      for (int32_t q = 0; q < per; ++q) {
        const int32_t ch = lane * per + q;
        ls += (ch < nchunks) ? chunk_mass[ch] : 0.f;
      }
      float incl = ls;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const float y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      const float Z = __shfl_sync(0xffffffffu, incl, 31);
      if (!(Z > 0.f)) {
        if (from_p && lane == 0) {  // no positive mass at all (non-finite logits)
          a.out_tok[r] = -1;
          record_status(a.status, SSD_ERR_DEVICE_BOUNDS);
        }
      } else {
        const float target = sh.u_res * Z;
        // lane holding the crossing (else the last lane with mass)
        const uint32_t pos = __ballot_sync(0xffffffffu, ls > 0.f);
        const uint32_t cross = __ballot_sync(0xffffffffu, ls > 0.f && incl > target);
        const int32_t ls_star = cross ? (__ffs(cross) - 1) : (31 - __clz(pos));
        float t1 = __shfl_sync(0xffffffffu, incl - ls, ls_star);
        t1 = cross ? target - t1 : INFINITY;
        // chunk inside that lane's range (same order as its sum)
        int32_t chs = -1, chlast = -1;
        float tch = INFINITY;
        if (lane == ls_star) {
          float cum = 0.f;
          for (int32_t q = 0; q < per; ++q) {
            const int32_t ch = lane * per + q;
            const float m = (ch < nchunks) ? chunk_mass[ch] : 0.f;
            if (m > 0.f) {
              chlast = ch;
              if (chs < 0 && cum + m > t1) { chs = ch; tch = t1 - cum; }
            }
            cum += m;
          }
          if (chs < 0) { chs = chlast; tch = INFINITY; }
        }
        chs = __shfl_sync(0xffffffffu, chs, ls_star);
        tch = __shfl_sync(0xffffffffu, tch, ls_star);
        // re-walk chunk chs = 8k + w: entries 4 * (k * 256 + w * 32 + lane) + 0..3
        const int32_t kk = chs / kWarps, ww = chs % kWarps;
        const int32_t i = kk * kThreads + ww * 32 + lane;
        float4 xp = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY), xq = xp;
        if (i < nv) {
          xp = ld_keep(tp + i);
          xq = from_p ? xp : ld_keep(dp + i);
        }
        const float4 w = weights4(xp, xq, c, Cp, Cq, from_p);
        const float lsum = (w.x + w.y) + (w.z + w.w);
        float li = lsum;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const float y = __shfl_up_sync(0xffffffffu, li, o);
          if (lane >= o) li += y;
        }
        const int32_t e = 4 * i;
        int32_t lp = -1;  // last entry of this lane with positive weight
        if (w.w > 0.f) lp = e + 3; else if (w.z > 0.f) lp = e + 2;
        else if (w.y > 0.f) lp = e + 1; else if (w.x > 0.f) lp = e;
        const uint32_t hasp = __ballot_sync(0xffffffffu, lp >= 0);
        const uint32_t lcross = __ballot_sync(0xffffffffu, lsum > 0.f && li > tch);
        const int32_t lstar = lcross ? (__ffs(lcross) - 1) : (hasp ? 31 - __clz(hasp) : 0);
        if (lane == lstar) {
          const float t4 = tch - (li - lsum);
          const float ws[4] = {w.x, w.y, w.z, w.w};
          float cc = 0.f;
          int32_t pick = -1;
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            cc += ws[k];
            if (pick < 0 && ws[k] > 0.f && cc > t4) pick = e + k;
          }
          if (pick < 0) pick = lp;
          a.out_tok[r] = pick;
        }
      }
      if (lane == 0) sh.accept = (Z > 0.f) ? 3 : 0;  // 3: drawn
    }
    __syncthreads();
    if (sh.accept == 3 || from_p) break;
  }
}

}  // namespace

bool accept_supported(int32_t V) { return V <= kMaxV; }

cudaError_t launch_accept(const AcceptArgs& a, cudaStream_t stream) {
  if (a.rows == 0) return cudaSuccess;
  const int32_t nv = a.V / 4;
  const int32_t iters = (nv + kThreads - 1) / kThreads;
  const size_t smem = (size_t)iters * kWarps * sizeof(float);
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(accept_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
  }
  accept_kernel<<<(unsigned)a.rows, kThreads, smem, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace ssd
