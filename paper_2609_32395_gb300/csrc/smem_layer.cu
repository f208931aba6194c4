// smem_layer.cu -- the dense parts of one reader layer around the attention
// path: LayerNorm, GELU and the projections (arXiv 2609.32395, Sec. 2
// "Model" and App. A "Reader": three pre-LN residual branches -- block-local
// causal self-attention, cross-attention into earlier blocks' memory rows,
// FFN of width 4d with GELU; memory rows are projected to each layer's keys
// and values, the null row likewise).
//
// The projections are plain GEMMs (bf16 operands, fp32 accumulation) and go
// to cuBLAS; everything else is a kernel here. Row-major [m][k] x [k][n]
// products map onto cuBLAS's column-major convention as C^T = B^T A^T.
// cuBLAS runs on a caller-provided workspace, so every call is stream-ordered
// and capturable in a CUDA graph; with a fixed workspace and shape its
// results are the same bits on every run.
#include <cublas_v2.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdio>

#include "smem_device.cuh"
#include "smem_internal.h"

namespace smem {

namespace {

constexpr int kRowThreads = 256;  // 8 warps, one row each

// h = LayerNorm(x) * g + b in fp32 (mean, then the biased variance of the
// centred values), rounded to bf16. x [n][d] fp32, d a multiple of 4.
__global__ void __launch_bounds__(kRowThreads) layernorm_kernel(const float* __restrict__ x, int n, int d,
                                                                 const float* __restrict__ g,
                                                                 const float* __restrict__ b, float eps,
                                                                 uint16_t* __restrict__ h) {
  const int lane = threadIdx.x & 31;
  const int row = blockIdx.x * (kRowThreads / 32) + (threadIdx.x >> 5);
  if (row >= n) return;
  const float4* xr = reinterpret_cast<const float4*>(x + (size_t)row * d);
  const int c4 = d / 4;
  float s = 0.f;
  for (int c = lane; c < c4; c += 32) {
    const float4 v = xr[c];
    s += (v.x + v.y) + (v.z + v.w);
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  const float mean = s / (float)d;
  float q = 0.f;
  for (int c = lane; c < c4; c += 32) {
    const float4 v = xr[c];
    const float a = v.x - mean, bb = v.y - mean, cc = v.z - mean, dd = v.w - mean;
    q += (a * a + bb * bb) + (cc * cc + dd * dd);
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) q += __shfl_xor_sync(0xffffffffu, q, o);
  const float rstd = rsqrtf(q / (float)d + eps);
  const float4* g4 = reinterpret_cast<const float4*>(g);
  const float4* b4 = reinterpret_cast<const float4*>(b);
  uint2* hr = reinterpret_cast<uint2*>(h + (size_t)row * d);
  for (int c = lane; c < c4; c += 32) {
    const float4 v = xr[c], gg = g4[c], bv = b4[c];
    uint2 o;
    o.x = pack_bf16x2((v.x - mean) * rstd * gg.x + bv.x, (v.y - mean) * rstd * gg.y + bv.y);
    o.y = pack_bf16x2((v.z - mean) * rstd * gg.z + bv.z, (v.w - mean) * rstd * gg.w + bv.w);
    hr[c] = o;
  }
}

__device__ __forceinline__ float gelu_erf(float v) { return 0.5f * v * (1.f + erff(v * 0.70710678118654752f)); }

// out = GELU(f) = f * Phi(f), rounded to bf16; n4 groups of 4 values.
__global__ void gelu_kernel(const float4* __restrict__ f, uint2* __restrict__ out, long long n4) {
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += (long long)gridDim.x * blockDim.x) {
    const float4 v = f[i];
    uint2 o;
    o.x = pack_bf16x2(gelu_erf(v.x), gelu_erf(v.y));
    o.y = pack_bf16x2(gelu_erf(v.z), gelu_erf(v.w));
    out[i] = o;
  }
}

inline cublasHandle_t handle(void* blas) { return static_cast<cublasHandle_t>(blas); }

int blas_status(cublasStatus_t s, const char* what, char* detail, size_t detail_len) {
  if (s == CUBLAS_STATUS_SUCCESS) return 0;
  std::snprintf(detail, detail_len, "%s: cuBLAS status %d", what, (int)s);
  return -1;
}

}  // namespace

cudaError_t launch_layernorm(const float* x, int n, int d, const float* g, const float* b, float eps, uint16_t* h,
                             cudaStream_t st) {
  if (n == 0) return cudaSuccess;
  const int rows_per_cta = kRowThreads / 32;
  layernorm_kernel<<<(n + rows_per_cta - 1) / rows_per_cta, kRowThreads, 0, st>>>(x, n, d, g, b, eps, h);
  return cudaGetLastError();
}

cudaError_t launch_gelu(const float* f, uint16_t* out, long long n, cudaStream_t st) {
  const long long n4 = n / 4;
  if (n4 == 0) return cudaSuccess;
  long long blocks = (n4 + 255) / 256;
  if (blocks > 2048) blocks = 2048;
  gelu_kernel<<<(int)blocks, 256, 0, st>>>(reinterpret_cast<const float4*>(f), reinterpret_cast<uint2*>(out), n4);
  return cudaGetLastError();
}

int blas_create(void** out, char* detail, size_t detail_len) {
  cublasHandle_t h = nullptr;
  if (blas_status(cublasCreate(&h), "cublasCreate", detail, detail_len)) return -1;
  *out = h;
  return 0;
}

void blas_destroy(void* blas) {
  if (blas) cublasDestroy(handle(blas));
}

int blas_bind(void* blas, cudaStream_t st, void* ws, size_t ws_bytes, char* detail, size_t detail_len) {
  if (blas_status(cublasSetStream(handle(blas), st), "cublasSetStream", detail, detail_len)) return -1;
  return blas_status(cublasSetWorkspace(handle(blas), ws, ws_bytes), "cublasSetWorkspace", detail, detail_len);
}

// C[m][n] (bf16, or fp32 with c_f32) = A[m][k] W[k][n] (+ C if accumulate),
// row-major, A and W bf16, fp32 accumulation.
int blas_gemm(void* blas, int m, int n, int k, const uint16_t* A, const uint16_t* W, void* C, bool c_f32,
              bool accumulate, char* detail, size_t detail_len) {
  if (m == 0) return 0;
  const float one = 1.f, zero = 0.f;
  return blas_status(cublasGemmEx(handle(blas), CUBLAS_OP_N, CUBLAS_OP_N, n, m, k, &one, W, CUDA_R_16BF, n, A,
                                  CUDA_R_16BF, k, accumulate ? &one : &zero, C, c_f32 ? CUDA_R_32F : CUDA_R_16BF, n,
                                  CUBLAS_COMPUTE_32F, CUBLAS_GEMM_DEFAULT),
                     "gemm", detail, detail_len);
}

// Per-head projection of rows: for every head h, out + h * head_stride holds
// [rows][D] = X[rows][d] W[:, h*D : (h+1)*D], bf16 (one batched GEMM); W is
// [d][ldw] row-major.
int blas_project_heads(void* blas, int rows, int d, int H, int D, const uint16_t* X, const uint16_t* W, int ldw,
                       uint16_t* out, long long head_stride, char* detail, size_t detail_len) {
  const float one = 1.f, zero = 0.f;
  return blas_status(cublasGemmStridedBatchedEx(handle(blas), CUBLAS_OP_N, CUBLAS_OP_N, D, rows, d, &one, W, CUDA_R_16BF,
                                                ldw, (long long)D, X, CUDA_R_16BF, d, 0LL, &zero, out, CUDA_R_16BF, D,
                                                head_stride, H, CUBLAS_COMPUTE_32F, CUBLAS_GEMM_DEFAULT),
                     "head projection", detail, detail_len);
}

// Column-major strided-batched GEMM (cuBLAS conventions), bf16 in and out,
// fp32 accumulation: C_i = alpha op(A_i) op(B_i), i < batch.
int blas_gemm_sb(void* blas, bool ta, bool tb, int m, int n, int k, float alpha, const uint16_t* A, int lda,
                 long long sA, const uint16_t* B, int ldb, long long sB, uint16_t* C, int ldc, long long sC, int batch,
                 char* detail, size_t detail_len) {
  if (m == 0 || n == 0) return 0;
  const float zero = 0.f;
  return blas_status(cublasGemmStridedBatchedEx(handle(blas), ta ? CUBLAS_OP_T : CUBLAS_OP_N,
                                                tb ? CUBLAS_OP_T : CUBLAS_OP_N, m, n, k, &alpha, A, CUDA_R_16BF, lda,
                                                sA, B, CUDA_R_16BF, ldb, sB, &zero, C, CUDA_R_16BF, ldc, sC, batch,
                                                CUBLAS_COMPUTE_32F, CUBLAS_GEMM_DEFAULT),
                     "batched gemm", detail, detail_len);
}

}  // namespace smem
