// probes.cu -- measurement probes for the roofline denominators: an FFMA
// chain (the FP32 pipe), a tanh.approx.f32 chain (the multi-function unit)
// and a cuBLAS GEMM in tf32 or bf16 (the tensor pipe for those operand
// types).  Each launches work of a known operation count on the caller's
// stream; the caller times it with events.  Not on any hot path.
#include <cublas_v2.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <mutex>

#include "auvenv.h"

namespace {

constexpr int kChains = 8;   // independent dependency chains per thread

// iters x kChains dependent FMAs per thread (2 flop each); the result is kept
// live through `sink` so that nothing is removed.
__global__ void k_probe_ffma(uint32_t iters, float* sink) {
  float a[kChains];
#pragma unroll
  for (int j = 0; j < kChains; ++j) a[j] = 1.0f + 1e-3f * (threadIdx.x + j);
  const float x = 0.9999f, y = 1e-4f;
  for (uint32_t i = 0; i < iters; ++i) {
#pragma unroll
    for (int j = 0; j < kChains; ++j) a[j] = fmaf(a[j], x, y);
  }
  float s = 0.0f;
#pragma unroll
  for (int j = 0; j < kChains; ++j) s += a[j];
  if (s == 12345.678f) sink[blockIdx.x * blockDim.x + threadIdx.x] = s;
}

// iters x kChains dependent tanh.approx.f32 per thread (one operation each).
__global__ void k_probe_tanh(uint32_t iters, float* sink) {
  float a[kChains];
#pragma unroll
  for (int j = 0; j < kChains; ++j) a[j] = 1e-3f * (threadIdx.x + j);
  for (uint32_t i = 0; i < iters; ++i) {
#pragma unroll
    for (int j = 0; j < kChains; ++j) {
      float r;
      asm("tanh.approx.f32 %0, %1;" : "=f"(r) : "f"(a[j]));
      a[j] = r + 0.5f;
    }
  }
  float s = 0.0f;
#pragma unroll
  for (int j = 0; j < kChains; ++j) s += a[j];
  if (s == 12345.678f) sink[blockIdx.x * blockDim.x + threadIdx.x] = s;
}

int probe_grid(uint32_t blocks, uint32_t threads, uint32_t iters, const float* sink) {
  if (blocks < 1 || blocks > 65535 || threads < 32 || threads > 1024 || threads % 32 || iters < 1 ||
      !sink)
    return AUV_ERR_INVALID;
  return AUV_OK;
}

std::mutex g_blas_mu;
cublasHandle_t g_blas = nullptr;

}  // namespace

extern "C" {

int auv_probe_ffma(uint32_t blocks, uint32_t threads, uint32_t iters, float* sink, void* stream) {
  int rc = probe_grid(blocks, threads, iters, sink);
  if (rc) return rc;
  k_probe_ffma<<<blocks, threads, 0, static_cast<cudaStream_t>(stream)>>>(iters, sink);
  return cudaGetLastError() == cudaSuccess ? AUV_OK : AUV_ERR_CUDA;
}

int auv_probe_tanh(uint32_t blocks, uint32_t threads, uint32_t iters, float* sink, void* stream) {
  int rc = probe_grid(blocks, threads, iters, sink);
  if (rc) return rc;
  k_probe_tanh<<<blocks, threads, 0, static_cast<cudaStream_t>(stream)>>>(iters, sink);
  return cudaGetLastError() == cudaSuccess ? AUV_OK : AUV_ERR_CUDA;
}

int auv_probe_gemm(uint32_t precision, int n, const void* a, const void* b, void* c, void* stream) {
  if (n < 16 || n % 16 || !a || !b || !c) return AUV_ERR_INVALID;
  if (precision != AUV_PPO_TF32 && precision != AUV_PPO_BF16) return AUV_ERR_INVALID;
  std::lock_guard<std::mutex> lock(g_blas_mu);
  if (!g_blas && cublasCreate(&g_blas) != CUBLAS_STATUS_SUCCESS) {
    g_blas = nullptr;
    return AUV_ERR_CUDA;
  }
  if (cublasSetStream(g_blas, static_cast<cudaStream_t>(stream)) != CUBLAS_STATUS_SUCCESS)
    return AUV_ERR_CUDA;
  const float one = 1.0f, zero = 0.0f;
  const bool tf32 = precision == AUV_PPO_TF32;
  const cudaDataType_t t = tf32 ? CUDA_R_32F : CUDA_R_16BF;
  const cublasStatus_t s =
      cublasGemmEx(g_blas, CUBLAS_OP_N, CUBLAS_OP_N, n, n, n, &one, a, t, n, b, t, n, &zero, c,
                   CUDA_R_32F, n, tf32 ? CUBLAS_COMPUTE_32F_FAST_TF32 : CUBLAS_COMPUTE_32F,
                   CUBLAS_GEMM_DEFAULT);
  return s == CUBLAS_STATUS_SUCCESS ? AUV_OK : AUV_ERR_CUDA;
}

}  // extern "C"
