// probes.cu -- measurement probes for the roofline denominators: an FFMA
// chain (the FP32 pipe), tanh.approx.f32 and ex2.approx.f32 chains (the
// multi-function unit), a cuBLAS GEMM in tf32 or bf16 (the tensor pipe for
// those operand types), and back-to-back tcgen05 MMAs of one shape (the
// tensor pipe's cost per instruction at the engine's small N).  Each
// launches work of a known operation count on the caller's stream; the
// caller times it with events (the MMA probe times itself in cycles).  Not
// on any hot path.
#include <cublas_v2.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <mutex>

#include "auvenv.h"
#include "tc_ptx.cuh"

namespace {

namespace tc = auv::tc;

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

// iters x kChains dependent ex2.approx.ftz.f32 per thread (one operation each).
__global__ void k_probe_ex2(uint32_t iters, float* sink) {
  float a[kChains];
#pragma unroll
  for (int j = 0; j < kChains; ++j) a[j] = 1e-3f * (threadIdx.x + j);
  for (uint32_t i = 0; i < iters; ++i) {
#pragma unroll
    for (int j = 0; j < kChains; ++j) {
      float r;
      asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(a[j]));
      a[j] = r - 1.0f;
    }
  }
  float s = 0.0f;
#pragma unroll
  for (int j = 0; j < kChains; ++j) s += a[j];
  if (s == 12345.678f) sink[blockIdx.x * blockDim.x + threadIdx.x] = s;
}

// kind::tf32 MMAs (D fp32, A and B tf32, K-major; K = 8 per instruction):
// instruction descriptor and the two operand forms.
__host__ __device__ constexpr uint32_t idesc_tf32_f32(int M, int N) {
  return (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(N >> 3) << 17) |
         ((uint32_t)(M >> 4) << 24);
}
__device__ __forceinline__ void mma_tf32_ss(uint32_t d, uint64_t a, uint64_t b, uint32_t id,
                                            uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}" ::"r"(d),
      "l"(a), "l"(b), "r"(id), "r"(acc)
      : "memory");
}
__device__ __forceinline__ void mma_tf32_ts(uint32_t d, uint32_t a, uint64_t b, uint32_t id,
                                            uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::tf32 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d),
      "r"(a), "l"(b), "r"(id), "r"(acc)
      : "memory");
}

// One elected thread per CTA issues `iters` tcgen05 MMAs of shape M = 128,
// N, K = 16 bf16 (kind::f16) or K = 8 tf32 (kind::tf32) operands,
// zero-filled, fp32 accumulator in tensor memory columns 0..N-1, back to back
// into one accumulator, with B from shared memory (128-byte swizzled K-major
// rows: one K-step is 32 bytes for either type) and A from shared memory or
// from tensor memory (columns 256..287), commits once and waits (bounded)
// for the completion.  cycles[block] = clock64 span from the first issue to
// the completion, or 0 if the wait gave up.  120 KB of shared memory keep
// one CTA per SM.
constexpr uint32_t kMmaSmem = 120u * 1024u;
template <int N, bool kTs, bool kTf32>
__global__ void __launch_bounds__(128) k_probe_mma(uint32_t iters, unsigned long long* cycles) {
  extern __shared__ uint8_t mma_smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(mma_smem_raw) + 1023u) & ~(uintptr_t)1023u);
  __shared__ uint64_t bar;
  __shared__ uint32_t tmem_base;
  __shared__ int abort_flag;
  const int tid = threadIdx.x;
  // operands: B at 0 (N rows x 128 B), A at 32 KB (128 rows x 128 B)
  for (int i = tid; i < 48 * 1024 / 16; i += 128)
    reinterpret_cast<uint4*>(smem)[i] = make_uint4(0u, 0u, 0u, 0u);
  if (tid == 0) {
    tc::mbar_init(&bar, 1);
    abort_flag = 0;
    tc::mbar_fence_init();
  }
  if (tid < 32) {
    tc::tmem_alloc(&tmem_base, 512);
    tc::tmem_relinquish();
  }
  tc::fence_async_smem();
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = tmem_base;
  if (tid == 0) {
    const uint32_t sb = tc::smem_u32(smem);
    const uint64_t b_desc = tc::smem_desc(sb, 1024, 2);
    const uint64_t a_desc = tc::smem_desc(sb + 32768, 1024, 2);
    constexpr uint32_t kIdesc = kTf32 ? idesc_tf32_f32(128, N) : tc::idesc_bf16_f32(128, N);
    const unsigned long long t0 = clock64();
    for (uint32_t i = 0; i < iters; ++i) {
      const uint32_t kk = i & 3u;   // the four 32-byte K-steps of a 128-byte row
      const uint32_t acc = i > 0 ? 1u : 0u;
      if constexpr (kTs && kTf32)
        mma_tf32_ts(tmem, tmem + 256 + kk * 8, b_desc + (uint64_t)(kk * 2), kIdesc, acc);
      else if constexpr (kTf32)
        mma_tf32_ss(tmem, a_desc + (uint64_t)(kk * 2), b_desc + (uint64_t)(kk * 2), kIdesc, acc);
      else if constexpr (kTs)
        tc::mma_ts(tmem, tmem + 256 + kk * 8, b_desc + (uint64_t)(kk * 2), kIdesc, acc);
      else
        tc::mma_ss(tmem, a_desc + (uint64_t)(kk * 2), b_desc + (uint64_t)(kk * 2), kIdesc, acc);
    }
    tc::mma_commit(&bar);
    const bool ok = tc::mbar_wait(&bar, 0, &abort_flag, 1000000000ull);
    cycles[blockIdx.x] = ok ? clock64() - t0 : 0ull;
  }
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  if (tid < 32) tc::tmem_dealloc(tmem, 512);
}

template <int N, bool kTs, bool kTf32>
cudaError_t launch_probe_mma(uint32_t iters, uint32_t blocks, unsigned long long* cycles,
                             cudaStream_t s) {
  cudaError_t e = cudaFuncSetAttribute(k_probe_mma<N, kTs, kTf32>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, kMmaSmem);
  if (e != cudaSuccess) return e;
  k_probe_mma<N, kTs, kTf32><<<blocks, 128, kMmaSmem, s>>>(iters, cycles);
  return cudaGetLastError();
}

template <bool kTs, bool kTf32>
cudaError_t launch_probe_mma_n(int n, uint32_t iters, uint32_t blocks, unsigned long long* cycles,
                               cudaStream_t s) {
  switch (n) {
    case 16: return launch_probe_mma<16, kTs, kTf32>(iters, blocks, cycles, s);
    case 32: return launch_probe_mma<32, kTs, kTf32>(iters, blocks, cycles, s);
    case 64: return launch_probe_mma<64, kTs, kTf32>(iters, blocks, cycles, s);
    case 128: return launch_probe_mma<128, kTs, kTf32>(iters, blocks, cycles, s);
    default: return launch_probe_mma<256, kTs, kTf32>(iters, blocks, cycles, s);
  }
}

// Device (or managed) memory on the current device: the probes write there
// from the GPU, so a host pointer is rejected before any launch.
bool device_ptr(const void* p) {
  cudaPointerAttributes a;
  int dev = -1;
  if (!p || cudaPointerGetAttributes(&a, p) != cudaSuccess || cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeManaged || (a.type == cudaMemoryTypeDevice && a.device == dev);
}

int probe_grid(uint32_t blocks, uint32_t threads, uint32_t iters, const float* sink) {
  if (blocks < 1 || blocks > 65535 || threads < 32 || threads > 1024 || threads % 32 || iters < 1 ||
      !device_ptr(sink))
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

int auv_probe_ex2(uint32_t blocks, uint32_t threads, uint32_t iters, float* sink, void* stream) {
  int rc = probe_grid(blocks, threads, iters, sink);
  if (rc) return rc;
  k_probe_ex2<<<blocks, threads, 0, static_cast<cudaStream_t>(stream)>>>(iters, sink);
  return cudaGetLastError() == cudaSuccess ? AUV_OK : AUV_ERR_CUDA;
}

int auv_probe_mma(int n, int a_tmem, int tf32, uint32_t iters, uint32_t blocks, uint64_t* cycles,
                  void* stream) {
  if ((n != 16 && n != 32 && n != 64 && n != 128 && n != 256) || iters < 1 || iters > (1u << 20) ||
      blocks < 1 || blocks > 65535 || !device_ptr(cycles))
    return AUV_ERR_INVALID;
  unsigned long long* c = reinterpret_cast<unsigned long long*>(cycles);
  const cudaStream_t s = static_cast<cudaStream_t>(stream);
  const cudaError_t e =
      tf32 ? (a_tmem ? launch_probe_mma_n<true, true>(n, iters, blocks, c, s)
                     : launch_probe_mma_n<false, true>(n, iters, blocks, c, s))
           : (a_tmem ? launch_probe_mma_n<true, false>(n, iters, blocks, c, s)
                     : launch_probe_mma_n<false, false>(n, iters, blocks, c, s));
  return e == cudaSuccess ? AUV_OK : AUV_ERR_CUDA;
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
