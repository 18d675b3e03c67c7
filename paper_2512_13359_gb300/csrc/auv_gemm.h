// auv_gemm.h -- dense products of the learners (PPO update, SHAC window) on the
// library's own kernels: tcgen05 tensor-core GEMMs (bf16 or tf32 operands,
// fp32 accumulation in tensor memory) and an fp32 CUDA-core GEMM.
//
//   C[M][N] = beta * C + sum_k A(m, k) B(n, k)            (row-major C, ldc)
//
// Each operand is either K-major (element (r, k) at r * ld + k: a row-major
// activation or weight array whose rows are the M or N index) or MN-major
// (element (r, k) at k * ld + r: a sample-major activation read along the
// batch, as in the weight gradients, whose contraction runs over samples).
// The tensor-core path loads 128-byte-swizzled tiles with TMA; operand
// addresses must be 16-byte aligned and ld * element size a multiple of 16.
// Contractions over the batch are split over CTAs (split-K) into fp32
// partials that a second kernel adds in a fixed order, so results do not
// depend on scheduling.
#pragma once

#include <cstddef>
#include <cstdint>

#include <cuda_runtime.h>

namespace auv {
struct Status;

namespace gemm {

enum Prec { kFp32 = 0, kTf32 = 1, kBf16 = 2 };   // the AUV_PPO_* precisions

struct Operand {
  const void* ptr;   // device memory: fp32 (kFp32, kTf32) or bf16 (kBf16) elements
  int ld;            // elements between consecutive stored rows
  bool mn_major;     // false: (r, k) at r*ld + k; true: (r, k) at k*ld + r
};

// Bytes of split-K partials a product of this shape may use (0: none).
size_t workspace_bytes(int M, int N, int K);

// Enqueue C = beta C + A B^T on s.  c_bf16: C holds bf16 (else fp32).
// ws / ws_bytes: scratch for split-K partials (may be null: no split).
// st: status block for device-side wait timeouts (AUV_ERR_TIMEOUT).
// Returns cudaSuccess, cudaErrorInvalidValue for an unsupported layout
// (misaligned operand), or the launch error.
cudaError_t launch(Prec prec, int M, int N, int K, const Operand& A, const Operand& B, void* C,
                   int ldc, bool c_bf16, float beta, float* ws, size_t ws_bytes, Status* st,
                   cudaStream_t s);

}  // namespace gemm
}  // namespace auv
