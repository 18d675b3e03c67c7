// mlp_fp32.cuh -- fp32 policy / value networks on CUDA cores, for both
// environment models (input width IN = 18 or 12).
#pragma once

#include <cuda_runtime.h>

namespace auv {

// ---------------------------------------------------------------------------
// fp32 networks on CUDA cores: tanh(W1 x + b1) -> tanh(W2 h + b2) -> W3 h + b3.
// Weights row-major [out][in] in global memory, read as warp-uniform loads
// (one L1 transaction per warp); the first hidden layer of this thread's env
// lives in its own shared-memory column hs[k * kTile] (conflict-free).  The
// second hidden layer is consumed unit by unit by the output layer, so it is
// never stored.
// ---------------------------------------------------------------------------
constexpr int kTile = 128;

template <int IN, int H, int OUT>
__device__ __forceinline__ void mlp_fp32(const float* __restrict__ w, const float x[IN],
                                         float* hs, float out[OUT]) {
  static_assert(IN % 2 == 0, "input width must be even (float2 rows)");
  const float* W1 = w;
  const float* b1 = W1 + H * IN;
  const float* W2 = b1 + H;
  const float* b2 = W2 + H * H;
  const float* W3 = b2 + H;
  const float* b3 = W3 + OUT * H;
  for (int j = 0; j < H; ++j) {
    float s = __ldg(b1 + j);
    const float2* row = reinterpret_cast<const float2*>(W1 + j * IN);
#pragma unroll
    for (int i2 = 0; i2 < IN / 2; ++i2) {
      const float2 wv = __ldg(row + i2);
      s = fmaf(wv.x, x[2 * i2], s);
      s = fmaf(wv.y, x[2 * i2 + 1], s);
    }
    hs[j * kTile] = tanhf(s);
  }
#pragma unroll
  for (int o = 0; o < OUT; ++o) out[o] = __ldg(b3 + o);
  for (int j = 0; j < H; ++j) {
    float s0 = __ldg(b2 + j), s1 = 0.0f;
    const float4* row = reinterpret_cast<const float4*>(W2 + (size_t)j * H);
#pragma unroll 8
    for (int k4 = 0; k4 < H / 4; ++k4) {
      const float4 wv = __ldg(row + k4);
      s0 = fmaf(wv.x, hs[(4 * k4 + 0) * kTile], s0);
      s1 = fmaf(wv.y, hs[(4 * k4 + 1) * kTile], s1);
      s0 = fmaf(wv.z, hs[(4 * k4 + 2) * kTile], s0);
      s1 = fmaf(wv.w, hs[(4 * k4 + 3) * kTile], s1);
    }
    const float h2 = tanhf(s0 + s1);
#pragma unroll
    for (int o = 0; o < OUT; ++o) out[o] = fmaf(__ldg(W3 + o * H + j), h2, out[o]);
  }
}

}  // namespace auv
