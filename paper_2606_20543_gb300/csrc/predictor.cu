// predictor.cu — the spatial draft predictor f_phi (Sec. 3.3 "Draft
// Prediction in Latent Space", Eq. 2) and the draft tokens it yields:
//
//   h_hat = W0 z + SwiGLU(RMSNorm(W0 z)),  z = [h ; e],
//   SwiGLU(x) = W2 (silu(W1 x) * W3 x),    t_hat = argmax GenHead(RMSNorm(h_hat)).
//
// Design (GB300): for one row of W grid columns the predictor is a chain of
// skinny products (rows <= a few hundred) that stream 268 MB of weights per
// head plus the 4096 x V GenHead, so it is bound by HBM, not by the tensor
// cores.  The four projections and the GenHead are plain GEMMs and run as
// cuBLAS bf16 GEMMs (fp32 accumulation on the tensor cores, fp32 outputs);
// everything between them is a kernel of this file (float4 accesses, several
// loads in flight per thread: these kernels are latency-bound at a few dozen
// rows), and the data flow needs no copies:
//   H  = W0 z                 GEMM into the caller's hidden-state buffer (fp32)
//   At = RMSNorm(H) * gamma1  rmsnorm_kernel (bf16, the next GEMM's input)
//   UV = At [W1 | W3]^T       two GEMMs into the halves of one fp32 buffer
//   G  = silu(U) * V          swiglu_kernel (bf16)
//   H  = H + G W2^T           GEMM with beta = 1: the residual in place
//   Hn = RMSNorm(H) * gamma2  rmsnorm_kernel (bf16)
//   L  = Hn W_head            GEMM (fp32 logits, rows x V)
//   t  = argmax L             argmax_kernel (lowest index on ties)
#include <cublas_v2.h>
#include <cuda_bf16.h>

#include <algorithm>

#include "kernels.cuh"

namespace ssd {

namespace {

constexpr int kNormThreads = 256;

__device__ __forceinline__ float block_sum(float v, float* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  v = warp_sum(v);
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float t = 0.f;
  if (warp == 0) {
    t = lane < (int)(blockDim.x >> 5) ? red[lane] : 0.f;
    t = warp_sum(t);
    if (lane == 0) red[0] = t;
  }
  __syncthreads();
  return red[0];
}

// One CTA per row: y = x / sqrt(mean(x^2) + eps) * gamma, rounded to bf16.
// float4 accesses, unrolled so that several loads are in flight (d % 4 == 0).
__global__ void __launch_bounds__(kNormThreads) rmsnorm_kernel(const float* __restrict__ x,
                                                               const float* __restrict__ gamma,
                                                               float eps, int32_t d,
                                                               __nv_bfloat16* __restrict__ y) {
  __shared__ float red[32];
  const float4* xr = reinterpret_cast<const float4*>(x + (int64_t)blockIdx.x * d);
  const float4* g4 = reinterpret_cast<const float4*>(gamma);
  uint2* yr = reinterpret_cast<uint2*>(y + (int64_t)blockIdx.x * d);
  const int32_t n4 = d >> 2;
  float ss = 0.f;
#pragma unroll 4
  for (int32_t i = threadIdx.x; i < n4; i += blockDim.x) {
    const float4 v = xr[i];
    ss += (v.x * v.x + v.y * v.y) + (v.z * v.z + v.w * v.w);
  }
  const float inv = 1.0f / sqrtf(block_sum(ss, red) / (float)d + eps);
#pragma unroll 4
  for (int32_t i = threadIdx.x; i < n4; i += blockDim.x) {
    const float4 v = xr[i], gm = g4[i];
    uint2 o;
    o.x = pack_bf16x2(v.x * inv * gm.x, v.y * inv * gm.y);
    o.y = pack_bf16x2(v.z * inv * gm.z, v.w * inv * gm.w);
    yr[i] = o;
  }
}

// g = silu(u) * v over rows x m; uv holds [u | v] per row (2m floats).
__global__ void swiglu_kernel(const float* __restrict__ uv, int32_t rows, int32_t m,
                              __nv_bfloat16* __restrict__ g) {
  const int64_t n = (int64_t)rows * m;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = i / m, j = i - r * m;
    const float u = uv[r * 2 * m + j], v = uv[r * 2 * m + m + j];
    g[i] = __float2bfloat16_rn(u / (1.0f + expf(-u)) * v);
  }
}

// One CTA per row: the first index of the maximum logit (V % 4 == 0; float4
// loads, unrolled so that several are in flight).
__global__ void __launch_bounds__(kNormThreads) argmax_kernel(const float* __restrict__ logits,
                                                              int32_t V,
                                                              int32_t* __restrict__ out_tok) {
  __shared__ float sv[32];
  __shared__ int32_t si[32];
  const float4* lr = reinterpret_cast<const float4*>(logits + (int64_t)blockIdx.x * V);
  float bv = -INFINITY;
  int32_t bi = 0x7fffffff;
#pragma unroll 4
  for (int32_t i = threadIdx.x; i < (V >> 2); i += blockDim.x) {
    const float4 v = lr[i];  // ascending index per thread: the first maximum is kept
    if (v.x > bv) { bv = v.x; bi = 4 * i; }
    if (v.y > bv) { bv = v.y; bi = 4 * i + 1; }
    if (v.z > bv) { bv = v.z; bi = 4 * i + 2; }
    if (v.w > bv) { bv = v.w; bi = 4 * i + 3; }
  }
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
    const int32_t oi = __shfl_xor_sync(0xffffffffu, bi, o);
    if (ov > bv || (ov == bv && oi < bi)) { bv = ov; bi = oi; }
  }
  if (lane == 0) { sv[warp] = bv; si[warp] = bi; }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 1; w < (int)(blockDim.x >> 5); ++w)
      if (sv[w] > bv || (sv[w] == bv && si[w] < bi)) { bv = sv[w]; bi = si[w]; }
    out_tok[blockIdx.x] = bi;
  }
}

// cuBLAS handle per device and host thread, created on first use.
constexpr int kMaxDevices = 64;
cublasStatus_t blas_handle(cublasHandle_t* out) {
  thread_local cublasHandle_t handles[kMaxDevices] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
    return CUBLAS_STATUS_NOT_INITIALIZED;
  if (handles[dev] == nullptr) {
    const cublasStatus_t s = cublasCreate(&handles[dev]);
    if (s != CUBLAS_STATUS_SUCCESS) return s;
  }
  *out = handles[dev];
  return CUBLAS_STATUS_SUCCESS;
}

size_t al256(size_t x) { return (x + 255) & ~size_t(255); }
constexpr size_t kBlasWorkspace = (size_t)32 << 20;

}  // namespace

size_t predictor_workspace(int32_t rows, int32_t d, int32_t m, int32_t V, bool own_hidden) {
  size_t b = al256(kBlasWorkspace);
  b += al256((size_t)rows * d * 2);       // At / Hn (bf16)
  b += al256((size_t)rows * 2 * m * 4);   // [U | V] (fp32)
  b += al256((size_t)rows * m * 2);       // G (bf16)
  b += al256((size_t)rows * V * 4);       // logits (fp32)
  if (own_hidden) b += al256((size_t)rows * d * 4);
  return b;
}

cudaError_t launch_predictor(const PredictorArgs& p, void* ws, size_t ws_bytes,
                             cudaStream_t stream) {
  if (ws_bytes < predictor_workspace(p.rows, p.d, p.m, p.V, p.out_hidden == nullptr))
    return cudaErrorInvalidValue;
  unsigned char* w = static_cast<unsigned char*>(ws);
  void* blas_ws = w;
  w += al256(kBlasWorkspace);
  __nv_bfloat16* nrm = reinterpret_cast<__nv_bfloat16*>(w);
  w += al256((size_t)p.rows * p.d * 2);
  float* uv = reinterpret_cast<float*>(w);
  w += al256((size_t)p.rows * 2 * p.m * 4);
  __nv_bfloat16* g = reinterpret_cast<__nv_bfloat16*>(w);
  w += al256((size_t)p.rows * p.m * 2);
  float* logits = reinterpret_cast<float*>(w);
  w += al256((size_t)p.rows * p.V * 4);
  float* H = p.out_hidden;
  if (H == nullptr) H = reinterpret_cast<float*>(w);

  const int32_t rows = p.rows, d = p.d, m = p.m;
  const int swg_blocks = (int)std::min<int64_t>(((int64_t)rows * m + 255) / 256,
                                                4 * (int64_t)device_sm_count());
  cublasHandle_t h;
  if (blas_handle(&h) != CUBLAS_STATUS_SUCCESS) return cudaErrorUnknown;
  if (cublasSetStream(h, stream) != CUBLAS_STATUS_SUCCESS ||
      cublasSetWorkspace(h, blas_ws, kBlasWorkspace) != CUBLAS_STATUS_SUCCESS)
    return cudaErrorUnknown;
  // Y[rows][N] (ld ldy) = (accumulate ? Y : 0) + X[rows][K] op(W); W [N][K]
  // (a linear layer's [out][in], as the column-major product Y^T = W X^T), or
  // [K][N] when w_kn
  auto product = [&](int32_t N, int32_t K, const void* x, const void* w, bool w_kn, float* y,
                     int32_t ldy, bool accumulate) -> cudaError_t {
    const float alpha = 1.0f, beta = accumulate ? 1.0f : 0.0f;
    const cublasStatus_t st =
        w_kn ? cublasGemmEx(h, CUBLAS_OP_N, CUBLAS_OP_N, N, rows, K, &alpha, w, CUDA_R_16BF, N, x,
                            CUDA_R_16BF, K, &beta, y, CUDA_R_32F, ldy, CUBLAS_COMPUTE_32F,
                            CUBLAS_GEMM_DEFAULT)
             : cublasGemmEx(h, CUBLAS_OP_T, CUBLAS_OP_N, N, rows, K, &alpha, w, CUDA_R_16BF, K, x,
                            CUDA_R_16BF, K, &beta, y, CUDA_R_32F, ldy, CUBLAS_COMPUTE_32F,
                            CUBLAS_GEMM_DEFAULT);
    return st == CUBLAS_STATUS_SUCCESS ? cudaSuccess : cudaErrorUnknown;
  };
  cudaError_t e;
  // H = W0 z
  if ((e = product(d, 2 * d, p.z, p.w0, false, H, d, false)) != cudaSuccess) return e;
  rmsnorm_kernel<<<rows, kNormThreads, 0, stream>>>(H, p.gamma1, p.eps, d, nrm);
  // [U | V] = At [W1 | W3]^T: two products into the halves of each row of uv
  if ((e = product(m, d, nrm, p.w1, false, uv, 2 * m, false)) != cudaSuccess) return e;
  if ((e = product(m, d, nrm, p.w3, false, uv + m, 2 * m, false)) != cudaSuccess) return e;
  swiglu_kernel<<<swg_blocks, 256, 0, stream>>>(uv, rows, m, g);
  // H = H + G W2^T (the residual)
  if ((e = product(d, m, g, p.w2, false, H, d, true)) != cudaSuccess) return e;
  rmsnorm_kernel<<<rows, kNormThreads, 0, stream>>>(H, p.gamma2, p.eps, d, nrm);
  // logits[rows][V] = Hn[rows][d] W_head[d][V]
  if ((e = product(p.V, d, nrm, p.w_head, true, logits, p.V, false)) != cudaSuccess) return e;
  argmax_kernel<<<rows, kNormThreads, 0, stream>>>(logits, p.V, p.out_tok);
  return cudaGetLastError();
}

}  // namespace ssd
