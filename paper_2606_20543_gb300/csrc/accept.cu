// accept.cu — vocabulary-wide acceptance (steps a3-a5): target/draft softmax,
// the ratio at the draft token, the accept decision and, on rejection, the
// residual draw (Sec. 3.3 "Verification as Auto Correction", strategy (C)):
//   accept t with probability min(p(t) / q(t), 1); otherwise draw from
//   [p - q]_+ / sum [p - q]_+ (inverse CDF in vocabulary order, one uniform).
//
// Design (GB300): one thread-block cluster per row.  CTA c of the cluster
// owns the vocabulary slice [c * S, c * S + S) and pulls its slice of both
// logit rows into shared memory with two bulk TMA copies, so every logit is
// read from HBM exactly once.  Per-CTA max / sum-exp / argmax partials are
// exchanged through distributed shared memory; every CTA combines them in
// rank order (identical results everywhere), takes the decision, and on a
// rejection computes its slice's residual mass from the resident slice.  A
// second exchange of the per-CTA masses locates the CTA holding the CDF
// crossing, which scans its slice (warp segments in vocabulary order).
#include <cooperative_groups.h>

#include "kernels.cuh"

namespace cg = cooperative_groups;

namespace ssd {

namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kMaxCluster = 8;
constexpr int kSliceTarget = 4096;     // elements per CTA when the cluster has room
constexpr int kSliceMax = 16384;       // 128 KB of shared memory for both rows
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

struct Partial {
  float max_p, sum_p;  // over this slice, sum of exp2((x - max) * c)
  float max_q, sum_q;
  float xq_t, xp_t;    // logits at the slice's candidate draft token
  int32_t t;           // candidate draft token (argmax q of the slice, or the given one), -1 if none
  float z;             // residual mass of the slice
};

struct Shared {
  Partial part;                 // this CTA's partial (read by the cluster)
  float red_f[kWarps * 4];
  int32_t red_i[kWarps];
  float warp_mass[kWarps];
  uint64_t bar;
  // decision broadcast
  float c_p, c_q;               // log2-domain normalisers: max * c + log2(sum)
  int32_t t;
  int32_t accept;
  float u_res;
};

__device__ __forceinline__ bool better_arg(float v, int32_t i, float bv, int32_t bi) {
  return v > bv || (v == bv && (uint32_t)i < (uint32_t)bi);
}

// Residual weight of one entry: [p - q]_+ (or p itself for the Z == 0 draw).
__device__ __forceinline__ float weight(float xp, float xq, float c, float c_p, float c_q,
                                        bool from_p) {
  const float pv = exp2f(fmaf(xp, c, -c_p));
  if (from_p) return pv;
  const float qv = exp2f(fmaf(xq, c, -c_q));
  return fmaxf(pv - qv, 0.0f);
}

// Mass of warp `w`'s segment of the slice, iterations of 128 entries
// (lane l holds entries 4l..4l+3 of the iteration), summed in a fixed order.
__device__ __forceinline__ float4 weights4(const float* sp, const float* sq, int32_t e, int32_t n,
                                           float c, float c_p, float c_q, bool from_p) {
  float4 w = make_float4(0.f, 0.f, 0.f, 0.f);
  if (e < n) {  // n % 4 == 0, so a vector is either fully inside or outside
    const float4 xp = *reinterpret_cast<const float4*>(sp + e);
    const float4 xq = *reinterpret_cast<const float4*>(sq + e);
    w.x = weight(xp.x, xq.x, c, c_p, c_q, from_p);
    w.y = weight(xp.y, xq.y, c, c_p, c_q, from_p);
    w.z = weight(xp.z, xq.z, c, c_p, c_q, from_p);
    w.w = weight(xp.w, xq.w, c, c_p, c_q, from_p);
  }
  return w;
}

__global__ void __launch_bounds__(kThreads)
accept_kernel(AcceptArgs a, int32_t slice, int32_t csize) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  float* sp = reinterpret_cast<float*>(smem_raw);
  float* sq = sp + slice;
  Shared& sh = *reinterpret_cast<Shared*>(sq + slice);

  const int32_t tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t r = blockIdx.x / csize;
  const int32_t rank = blockIdx.x % csize;
  const bool lead = (rank == 0) && (tid == 0);

  // ---- rows outside the frontier (padding slots of a verification step)
  if (a.n_drafts != nullptr) {
    const int32_t b = (int32_t)(r / a.D_max), j = (int32_t)(r % a.D_max);
    if (j >= a.n_drafts[b]) {
      if (lead) {
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
      if (lead) {
        record_status(a.status, SSD_ERR_DEVICE_BOUNDS);
        a.out_tok[r] = -1;
        a.accepted[r] = 0;
        if (a.ratio) a.ratio[r] = 0.f;
      }
      return;
    }
  }

  const int32_t v0 = rank * slice;
  const int32_t n = min(slice, a.V - v0);  // > 0 by construction, multiple of 4

  // ---- stage the slice of both rows in shared memory (one HBM read)
  if (tid == 0) {
    mbar_init(&sh.bar, 1);
    fence_barrier_init();
  }
  __syncthreads();
  if (tid == 0) {
    const uint32_t bytes = (uint32_t)n * 4u;
    mbar_arrive_expect_tx(&sh.bar, 2u * bytes);
    bulk_g2s(sp, a.tgt + r * a.ld + v0, bytes, &sh.bar);
    bulk_g2s(sq, a.drf + r * a.ld + v0, bytes, &sh.bar);
  }
  const bool ok = mbar_wait(&sh.bar, 0, a.status);

  cg::cluster_group cluster = cg::this_cluster();
  const float c = kLog2e / a.temperature;

  // ---- pass 1: max of both rows, argmax of the draft row
  float mp = -INFINITY, mq = -INFINITY;
  int32_t iq = 0x7fffffff;
  const int32_t nv = n >> 2;
  if (ok) {
    for (int32_t i = tid; i < nv; i += kThreads) {
      const float4 xp = reinterpret_cast<const float4*>(sp)[i];
      const float4 xq = reinterpret_cast<const float4*>(sq)[i];
      mp = fmaxf(mp, fmaxf(fmaxf(xp.x, xp.y), fmaxf(xp.z, xp.w)));
      const int32_t e = v0 + 4 * i;
      if (better_arg(xq.x, e, mq, iq)) { mq = xq.x; iq = e; }
      if (better_arg(xq.y, e + 1, mq, iq)) { mq = xq.y; iq = e + 1; }
      if (better_arg(xq.z, e + 2, mq, iq)) { mq = xq.z; iq = e + 2; }
      if (better_arg(xq.w, e + 3, mq, iq)) { mq = xq.w; iq = e + 3; }
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    mp = fmaxf(mp, __shfl_xor_sync(0xffffffffu, mp, o));
    const float oq = __shfl_xor_sync(0xffffffffu, mq, o);
    const int32_t oi = __shfl_xor_sync(0xffffffffu, iq, o);
    if (better_arg(oq, oi, mq, iq)) { mq = oq; iq = oi; }
  }
  if (lane == 0) {
    sh.red_f[warp] = mp;
    sh.red_f[kWarps + warp] = mq;
    sh.red_i[warp] = iq;
  }
  __syncthreads();
  mp = sh.red_f[0];
  mq = sh.red_f[kWarps];
  iq = sh.red_i[0];
  for (int w = 1; w < kWarps; ++w) {
    mp = fmaxf(mp, sh.red_f[w]);
    if (better_arg(sh.red_f[kWarps + w], sh.red_i[w], mq, iq)) {
      mq = sh.red_f[kWarps + w];
      iq = sh.red_i[w];
    }
  }
  __syncthreads();

  // ---- pass 2: sum of exp relative to the slice maxima
  float s_p = 0.f, s_q = 0.f;
  if (ok) {
    const float mpc = mp * c, mqc = mq * c;
    for (int32_t i = tid; i < nv; i += kThreads) {
      const float4 xp = reinterpret_cast<const float4*>(sp)[i];
      const float4 xq = reinterpret_cast<const float4*>(sq)[i];
      s_p += exp2f(fmaf(xp.x, c, -mpc)) + exp2f(fmaf(xp.y, c, -mpc)) +
             exp2f(fmaf(xp.z, c, -mpc)) + exp2f(fmaf(xp.w, c, -mpc));
      s_q += exp2f(fmaf(xq.x, c, -mqc)) + exp2f(fmaf(xq.y, c, -mqc)) +
             exp2f(fmaf(xq.z, c, -mqc)) + exp2f(fmaf(xq.w, c, -mqc));
    }
  }
  s_p = warp_sum(s_p);
  s_q = warp_sum(s_q);
  if (lane == 0) {
    sh.red_f[2 * kWarps + warp] = s_p;
    sh.red_f[3 * kWarps + warp] = s_q;
  }
  __syncthreads();
  if (tid == 0) {
    float tp = 0.f, tq = 0.f;
    for (int w = 0; w < kWarps; ++w) {
      tp += sh.red_f[2 * kWarps + w];
      tq += sh.red_f[3 * kWarps + w];
    }
    Partial& P = sh.part;
    P.max_p = mp;
    P.sum_p = tp;
    P.max_q = mq;
    P.sum_q = tq;
    if (given_t >= 0) {
      const bool mine = given_t >= v0 && given_t < v0 + n;
      P.t = mine ? given_t : -1;
      P.xp_t = mine ? sp[given_t - v0] : 0.f;
      P.xq_t = mine ? sq[given_t - v0] : 0.f;
    } else if (ok && iq >= v0 && iq < v0 + n) {
      P.t = iq;
      P.xq_t = mq;
      P.xp_t = sp[iq - v0];
    } else {  // no finite candidate in this slice (NaN logits or a failed copy)
      P.t = -1;
      P.xq_t = -INFINITY;
      P.xp_t = 0.f;
    }
    P.z = 0.f;
  }
  if (csize > 1) cluster.sync(); else __syncthreads();

  // ---- combine the cluster's partials in rank order, decide (thread 0)
  if (tid == 0) {
    float Mp = -INFINITY, Mq = -INFINITY;
    for (int k = 0; k < csize; ++k) {
      const Partial* P = cluster.map_shared_rank(&sh.part, k);
      Mp = fmaxf(Mp, P->max_p);
      Mq = fmaxf(Mq, P->max_q);
    }
    float Sp = 0.f, Sq = 0.f, xp_t = 0.f, xq_t = -INFINITY;
    int32_t t = given_t >= 0 ? given_t : 0x7fffffff;
    for (int k = 0; k < csize; ++k) {
      const Partial* P = cluster.map_shared_rank(&sh.part, k);
      Sp += P->sum_p * exp2f((P->max_p - Mp) * c);
      Sq += P->sum_q * exp2f((P->max_q - Mq) * c);
      if (given_t >= 0) {
        if (P->t == given_t) { xp_t = P->xp_t; xq_t = P->xq_t; }
      } else if (better_arg(P->xq_t, P->t, xq_t, t)) {
        t = P->t;
        xq_t = P->xq_t;
        xp_t = P->xp_t;
      }
    }
    const bool valid_t = (t >= 0 && t < a.V);
    if (!valid_t) {
      record_status(a.status, SSD_ERR_DEVICE_BOUNDS);
      t = -1;
    }
    const float l2p = (xp_t - Mp) * c - log2f(Sp);
    const float l2q = (xq_t - Mq) * c - log2f(Sq);
    const float ratio = exp2f(l2p - l2q);
    const float2 u = row_uniforms(a.rng, r);
    const bool acc = valid_t && u.x < fminf(ratio, 1.0f);
    sh.t = t;
    sh.accept = acc ? 1 : (valid_t ? 0 : 2);  // 2: no valid draft token, skip the draw
    sh.c_p = Mp * c + log2f(Sp);
    sh.c_q = Mq * c + log2f(Sq);
    sh.u_res = u.y;
    if (rank == 0) {
      a.accepted[r] = acc ? 1 : 0;
      if (acc || !valid_t) a.out_tok[r] = t;
      if (a.ratio) a.ratio[r] = ratio;
      if (a.lse) {
        a.lse[2 * r] = Mp / a.temperature + log2f(Sp) * kLn2;
        a.lse[2 * r + 1] = Mq / a.temperature + log2f(Sq) * kLn2;
      }
    }
  }
  __syncthreads();

  if (sh.accept == 0) {
    // ---- residual draw: [p - q]_+ (or p when that mass is zero)
    const float c_p = sh.c_p, c_q = sh.c_q;
    const int32_t wseg = ((n + kWarps * 128 - 1) / (kWarps * 128)) * 128;  // per-warp entries
    const int32_t w_begin = warp * wseg;
    const int32_t iters = wseg / 128;
    for (int pass = 0; pass < 2; ++pass) {
      const bool from_p = (pass == 1);
      // R1: per-warp masses, fixed summation order (lane sums -> warp tree -> iterations)
      float mass = 0.f;
      if (ok) {
        for (int32_t it = 0; it < iters; ++it) {
          const float4 w = weights4(sp, sq, w_begin + it * 128 + 4 * lane, n, c, c_p, c_q, from_p);
          mass += warp_sum((w.x + w.y) + (w.z + w.w));
        }
      }
      if (lane == 0) sh.warp_mass[warp] = mass;
      __syncthreads();
      if (tid == 0) {
        float z = 0.f;
        for (int w = 0; w < kWarps; ++w) z += sh.warp_mass[w];
        sh.part.z = z;
      }
      if (csize > 1) cluster.sync(); else __syncthreads();
      // every thread reads the cluster's masses in rank order
      float Z = 0.f;
      for (int k = 0; k < csize; ++k) Z += cluster.map_shared_rank(&sh.part, k)->z;
      if (!(Z > 0.f) && !from_p) {
        if (csize > 1) cluster.sync(); else __syncthreads();  // everyone has read z
        continue;  // zero residual mass: draw from p instead
      }
      const float target = sh.u_res * Z;
      // locate the CTA holding the crossing
      int32_t cstar = -1, clast = -1;
      float tc = 0.f, cum = 0.f;
      for (int k = 0; k < csize; ++k) {
        const float zk = cluster.map_shared_rank(&sh.part, k)->z;
        if (zk > 0.f) {
          clast = k;
          if (cstar < 0 && cum + zk > target) { cstar = k; tc = target - cum; }
        }
        cum += zk;
      }
      if (clast < 0) {  // no positive mass anywhere (non-finite logits)
        if (rank == 0 && tid == 0) {
          a.out_tok[r] = -1;
          record_status(a.status, SSD_ERR_DEVICE_BOUNDS);
        }
        break;
      }
      if (cstar < 0) { cstar = clast; tc = INFINITY; }  // rounding ran past the end
      if (rank == cstar && ok) {
        // locate the warp segment
        int32_t wstar = -1, wlast = -1;
        float tw = 0.f, cw = 0.f;
        for (int w = 0; w < kWarps; ++w) {
          const float mw = sh.warp_mass[w];
          if (mw > 0.f) {
            wlast = w;
            if (wstar < 0 && cw + mw > tc) { wstar = w; tw = tc - cw; }
          }
          cw += mw;
        }
        if (wstar < 0) { wstar = wlast; tw = INFINITY; }
        if (warp == wstar) {
          // re-walk the segment with the same arithmetic as R1
          float run = 0.f;
          int32_t found = -1, last_pos = -1;
          for (int32_t it = 0; it < iters && found < 0; ++it) {
            const int32_t e = w_begin + it * 128 + 4 * lane;
            const float4 w = weights4(sp, sq, e, n, c, c_p, c_q, from_p);
            const float lsum = (w.x + w.y) + (w.z + w.w);
            const float isum = warp_sum(lsum);
            // last entry with positive weight so far (fallback)
            int32_t lp = -1;
            if (w.w > 0.f) lp = e + 3; else if (w.z > 0.f) lp = e + 2;
            else if (w.y > 0.f) lp = e + 1; else if (w.x > 0.f) lp = e;
            const uint32_t hasp = __ballot_sync(0xffffffffu, lp >= 0);
            if (hasp) last_pos = __shfl_sync(0xffffffffu, lp, 31 - __clz(hasp));
            if (isum > 0.f && run + isum > tw) {
              const float t3 = tw - run;
              // inclusive scan of lane sums in lane order
              float incl = lsum;
#pragma unroll
              for (int o = 1; o < 32; o <<= 1) {
                const float y = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl += y;
              }
              const float excl = incl - lsum;
              const uint32_t cross = __ballot_sync(0xffffffffu, lsum > 0.f && incl > t3);
              int32_t lstar = cross ? (__ffs(cross) - 1) : (31 - __clz(hasp));
              int32_t pick = -1;
              if (lane == lstar) {
                const float t4 = t3 - excl;
                float cc = 0.f;
                const float ws[4] = {w.x, w.y, w.z, w.w};
                for (int k = 0; k < 4 && pick < 0; ++k) {
                  cc += ws[k];
                  if (ws[k] > 0.f && cc > t4) pick = e + k;
                }
                if (pick < 0) pick = lp;  // last positive entry of this lane
              }
              found = __shfl_sync(0xffffffffu, pick, lstar);
            }
            run += isum;
          }
          if (found < 0) found = last_pos;
          if (lane == 0) a.out_tok[r] = v0 + found;
        }
      }
      break;
    }
  }
  // keep this CTA's shared memory alive until every peer finished reading it
  if (csize > 1) cluster.sync();
}

int pick_cluster(int32_t V, int32_t* slice_out) {
  int cs = (V + kSliceTarget - 1) / kSliceTarget;
  if (cs > kMaxCluster) cs = kMaxCluster;
  if (cs < 1) cs = 1;
  int32_t slice = (V + cs - 1) / cs;
  slice = (slice + 3) & ~3;
  *slice_out = slice;
  return cs;
}

}  // namespace

bool accept_supported(int32_t V) {
  int32_t slice;
  pick_cluster(V, &slice);
  return slice <= kSliceMax;
}

cudaError_t launch_accept(const AcceptArgs& a, cudaStream_t stream) {
  if (a.rows == 0) return cudaSuccess;
  int32_t slice;
  const int cs = pick_cluster(a.V, &slice);
  const size_t smem = (size_t)slice * 8 + sizeof(Shared) + 16;
  cudaError_t e = cudaFuncSetAttribute(accept_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)((int64_t)a.rows * cs), 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cs;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, accept_kernel, a, slice, (int32_t)cs);
}

}  // namespace ssd
