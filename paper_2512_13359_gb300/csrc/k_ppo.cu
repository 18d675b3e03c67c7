// k_ppo.cu -- on-GPU pieces of the PPO learner that consume the rollout's
// SoA trajectory (paper §III-A: PPO, Schulman et al. 2017).
//
// Generalised advantage estimation (Schulman et al. 2016) over [T][N]
// arrays, one thread per env walking t = T-1 .. 0:
//   delta_t = r_t + gamma (1 - d_t) V_{t+1} - V_t,   V_T = last_value
//   A_t = delta_t + gamma lambda (1 - d_t) A_{t+1};  R_t = A_t + V_t.
// The kernel is bound by HBM: 17 bytes per env-step (reward, done, value in;
// advantage, return out).  Each thread loads a block of kU steps before it
// runs their recursion, so that every warp keeps 3 kU coalesced loads in
// flight (16-step blocks: 3.1 TB/s at 65,536 envs x 128 steps, 4.3 TB/s at
// 262,144; 8- and 32-step blocks measured slower).
#include <cuda_bf16.h>

#include "auv_kernels.h"

namespace auv {

namespace {

constexpr int kU = 16;

__global__ void __launch_bounds__(256) k_gae(int n, int T, const float* __restrict__ rew,
                                             const uint8_t* __restrict__ done,
                                             const float* __restrict__ value,
                                             const float* __restrict__ last_value, float gamma,
                                             float gl, float* __restrict__ adv,
                                             float* __restrict__ ret) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const size_t N = (size_t)n;
  float a_next = 0.0f;
  float v_next = __ldg(last_value + i);
  for (int hi = T; hi > 0; hi -= kU) {
    const int cnt = hi < kU ? hi : kU;
    const int lo = hi - cnt;
    float r[kU], v[kU], nt[kU];
#pragma unroll
    for (int k = 0; k < kU; ++k) {
      if (k < cnt) {
        const size_t o = (size_t)(lo + k) * N + i;
        r[k] = __ldg(rew + o);
        v[k] = __ldg(value + o);
        nt[k] = __ldg(done + o) ? 0.0f : 1.0f;
      }
    }
#pragma unroll
    for (int k = kU - 1; k >= 0; --k) {
      if (k < cnt) {
        const float delta = fmaf(gamma * nt[k], v_next, r[k]) - v[k];
        a_next = fmaf(gl * nt[k], a_next, delta);
        const size_t o = (size_t)(lo + k) * N + i;
        adv[o] = a_next;
        ret[o] = a_next + v[k];
        v_next = v[k];
      }
    }
  }
}

// The same recursion split over C time chunks of L <= LC steps: warp c
// of a block runs chunk c for 32 envs (coalesced loads).  Pass one goes
// backwards over the chunk from a zero carry and keeps only the chunk's
// (A', P): its advantage at the chunk start given zero advantage after the
// chunk, and the product of gamma lambda (1 - d_t) over it, so that the true
// start value is A' + P A_next.  The block combines those in shared memory
// to the true advantage just after each chunk, and pass two reruns the
// chunk's recursion from it.  C times more threads than k_gae; 8-step chunks
// keep 48 warps resident per SM, 16-step ones 32.
template <int C, int LC>
__global__ void __launch_bounds__(32 * C, (LC <= 8 ? 48 : 32) / C) k_gae_chunked(int n, int T, const float* __restrict__ rew,
                                                        const uint8_t* __restrict__ done,
                                                        const float* __restrict__ value,
                                                        const float* __restrict__ last_value,
                                                        float gamma, float gl,
                                                        float* __restrict__ adv,
                                                        float* __restrict__ ret) {
  __shared__ float sA[C][32], sP[C][32];
  const int lane = threadIdx.x & 31, c = threadIdx.x >> 5;
  const int i = blockIdx.x * 32 + lane;
  const int L = (T + C - 1) / C;
  const int lo = c * L, hi = min(T, lo + L);
  const size_t N = (size_t)n;
  float dl[LC], v[LC];
  unsigned live_bits = 0;        // bit k: step lo + k is not an episode end
  float a = 0.0f, p = 1.0f;
  const bool live = i < n && lo < hi;
  if (live) {
    float r[LC];
    unsigned char d[LC];
#pragma unroll
    for (int k = 0; k < LC; ++k) {
      if (lo + k < hi) {
        const size_t o = (size_t)(lo + k) * N + i;
        r[k] = __ldg(rew + o);
        v[k] = __ldg(value + o);
        d[k] = __ldg(done + o);
      }
    }
    float v_next = hi == T ? __ldg(last_value + i) : __ldg(value + (size_t)hi * N + i);
#pragma unroll
    for (int k = LC - 1; k >= 0; --k) {
      if (lo + k < hi) {
        const float nt = d[k] ? 0.0f : 1.0f;
        live_bits |= d[k] ? 0u : 1u << k;
        dl[k] = fmaf(gamma * nt, v_next, r[k]) - v[k];
        a = fmaf(gl * nt, a, dl[k]);
        p *= gl * nt;
        v_next = v[k];
      }
    }
  }
  sA[c][lane] = a;      // an empty chunk is the identity (0, 1)
  sP[c][lane] = p;
  __syncthreads();
  if (!live) return;
  a = 0.0f;
  for (int c2 = C - 1; c2 > c; --c2) a = fmaf(sP[c2][lane], a, sA[c2][lane]);
#pragma unroll
  for (int k = LC - 1; k >= 0; --k) {
    if (lo + k < hi) {
      a = fmaf((live_bits >> k & 1u) ? gl : 0.0f, a, dl[k]);
      const size_t o = (size_t)(lo + k) * N + i;
      adv[o] = a;
      ret[o] = a + v[k];
    }
  }
}

}  // namespace

cudaError_t launch_gae(int n, int T, const float* rew, const uint8_t* done, const float* value,
                       const float* last_value, float gamma, float lam, float* adv, float* ret,
                       cudaStream_t s) {
  const float gl = gamma * lam;
  const unsigned nb = (unsigned)((n + 31) / 32);
#define AUV_GAE_CHUNKED(C, LC) \
  k_gae_chunked<C, LC><<<nb, 32 * C, 0, s>>>(n, T, rew, done, value, last_value, gamma, gl, adv, ret)
  // 8-step chunks up to T = 128 (C <= 16), 16-step ones up to T = 512
  if (T > 8 && T <= 512) {
    if (T <= 16) AUV_GAE_CHUNKED(2, 8);
    else if (T <= 32) AUV_GAE_CHUNKED(4, 8);
    else if (T <= 64) AUV_GAE_CHUNKED(8, 8);
    else if (T <= 128) AUV_GAE_CHUNKED(16, 8);
    else if (T <= 256) AUV_GAE_CHUNKED(16, 16);
    else AUV_GAE_CHUNKED(32, 16);
#undef AUV_GAE_CHUNKED
    return cudaGetLastError();
  }
  k_gae<<<(n + 255) / 256, 256, 0, s>>>(n, T, rew, done, value, last_value, gamma, gl, adv, ret);
  return cudaGetLastError();
}

}  // namespace auv

// ---------------------------------------------------------------------------
// PPO minibatch update (Schulman et al. 2017).  The GEMMs of the two MLPs run
// in k_gemm.cu and the tcgen05 engine; these kernels do everything around them: the
// epoch permutation and minibatch gather, tanh forward and backward, the
// per-sample loss and its gradient at the heads, the minibatch statistics,
// the global gradient norm and Adam, and the weight-layout conversion.
// ---------------------------------------------------------------------------
namespace auv {
namespace ppo {

namespace {

constexpr int kT = 256;
constexpr float kHalfLog2Pi = 0.91893853320467274f;

// Activation storage: fp32, or bf16 (round to nearest even) in bf16 mode.
__device__ __forceinline__ void st_act(float* p, float x) { *p = x; }
__device__ __forceinline__ void st_act(__nv_bfloat16* p, float x) { *p = __float2bfloat16_rn(x); }

// Balanced Feistel network, four rounds; round j: (L, R) -> (R, L ^ F_j(R)),
// F_j(R) = first Philox4x32-10 word at counter (R, j, epoch) and key seed.
__device__ __forceinline__ uint32_t feistel(uint32_t x, const PermKey& p) {
  uint32_t left = x >> p.h, right = x & p.mask;
#pragma unroll 1
  for (uint32_t j = 0; j < 4; ++j) {
    const uint4 o = philox10(right, j, p.e0, p.e1, p.k0, p.k1);
    const uint32_t next = left ^ (o.x & p.mask);
    left = right;
    right = next;
  }
  return (left << p.h) | right;
}

// Position j of the epoch's permutation of [0, m): cycle-walk the network
// until it lands inside (it returns to j at the latest, so this ends).
__device__ __forceinline__ uint32_t perm_index(uint32_t j, const PermKey& p) {
  uint32_t x = feistel(j, p);
  while (x >= p.m) x = feistel(x, p);
  return x;
}

// Sum NV values over the block (blockDim.x = kT); the result is in thread 0.
template <int NV, typename V>
__device__ __forceinline__ void block_sum(V (&v)[NV], V* sh /* [NV][kT/32] */) {
#pragma unroll
  for (int k = 0; k < NV; ++k)
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v[k] += __shfl_down_sync(0xFFFFFFFFu, v[k], o);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  if (l == 0)
#pragma unroll
    for (int k = 0; k < NV; ++k) sh[k * (kT / 32) + w] = v[k];
  __syncthreads();
  if (w == 0) {
#pragma unroll
    for (int k = 0; k < NV; ++k) {
      v[k] = l < kT / 32 ? sh[k * (kT / 32) + l] : V(0);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) v[k] += __shfl_down_sync(0xFFFFFFFFu, v[k], o);
    }
  }
  __syncthreads();
}

template <typename TX>
__global__ void __launch_bounds__(kT) k_gather(Dims d, PermKey key, const StepCtl* ctl,
                                               const float* __restrict__ obs,
                                               const float* __restrict__ act,
                                               const float* __restrict__ logp,
                                               const float* __restrict__ adv,
                                               const float* __restrict__ ret, uint32_t N,
                                               Sample out, TX* __restrict__ X) {
  __shared__ double sh[2 * (kT / 32)];
  const int b = blockIdx.x * kT + threadIdx.x;
  const unsigned long long epoch = ctl->epoch0 + ctl->step / ctl->n_mb;
  const uint32_t start = (ctl->step % ctl->n_mb) * (uint32_t)d.B;
  key.e0 = (uint32_t)epoch;
  key.e1 = (uint32_t)(epoch >> 32);
  double s[2] = {0.0, 0.0};
  if (b < d.B) {
    const uint32_t r = perm_index(start + (uint32_t)b, key);
    const size_t t = r / N, i = r - (uint32_t)t * N, n = N;
    TX* x = X + (size_t)b * d.Dp;
    // loads in chunks of 8 so that several are in flight per thread
    for (int k0 = 0; k0 < d.D; k0 += 8) {
      float v[8];
#pragma unroll
      for (int j = 0; j < 8; ++j)
        if (k0 + j < d.D) v[j] = __ldg(obs + (t * d.D + k0 + j) * n + i);
#pragma unroll
      for (int j = 0; j < 8; ++j)
        if (k0 + j < d.D) st_act(x + k0 + j, v[j]);
    }
    st_act(x + d.D, 1.0f);
    for (int k = d.D + 1; k < d.Dp; ++k) st_act(x + k, 0.0f);
    const size_t o = t * n + i;
    out.ret[b] = __ldg(ret + o);
    if (!d.value_only) {
      float av[8];
#pragma unroll
      for (int k = 0; k < 8; ++k)
        if (k < d.A) av[k] = __ldg(act + (t * d.A + k) * n + i);
#pragma unroll
      for (int k = 0; k < 8; ++k)
        if (k < d.A) out.act[(size_t)b * d.A + k] = av[k];
      const float a = __ldg(adv + o);
      out.logp[b] = __ldg(logp + o);
      out.adv[b] = a;
      s[0] = a;
      s[1] = (double)a * a;
    }
  }
  block_sum<2>(s, sh);
  if (threadIdx.x == 0) {
    out.adv_part[2 * blockIdx.x] = s[0];
    out.adv_part[2 * blockIdx.x + 1] = s[1];
  }
}

// Sample-major copy of a batch: row r = t N + i holds, in Ws floats (Ws a
// multiple of 8), obs[t][0..D), act[t][0..A), logp, adv, ret of (t, i), the
// rest zero.  A block transposes 32 consecutive envs of one step through
// shared memory: coalesced feature-major reads, one contiguous row-block
// write.  Absent arrays (value-only batches) read as zero.
constexpr int kSmRows = 32;
constexpr int kSmMaxW = 80;   // round8(64 + 8 + 3)

__global__ void __launch_bounds__(256) k_transpose_batch(int D, int A, int Ws, uint32_t N,
                                                         const float* __restrict__ obs,
                                                         const float* __restrict__ act,
                                                         const float* __restrict__ logp,
                                                         const float* __restrict__ adv,
                                                         const float* __restrict__ ret,
                                                         float* __restrict__ dst) {
  __shared__ float tile[kSmRows][kSmMaxW + 1];
  const uint32_t blocks_per_t = (N + kSmRows - 1) / kSmRows;
  const size_t t = blockIdx.x / blocks_per_t;
  const uint32_t i0 = (blockIdx.x % blocks_per_t) * kSmRows;
  const int F = D + A + 3;
  const size_t n = N;
  for (int e = threadIdx.x; e < F * kSmRows; e += blockDim.x) {
    const int f = e / kSmRows, row = e % kSmRows;
    const uint32_t i = i0 + row;
    float v = 0.0f;
    if (i < N) {
      if (f < D) v = __ldg(obs + (t * D + f) * n + i);
      else if (f < D + A) v = act ? __ldg(act + (t * A + (f - D)) * n + i) : 0.0f;
      else if (f == D + A) v = logp ? __ldg(logp + t * n + i) : 0.0f;
      else if (f == D + A + 1) v = adv ? __ldg(adv + t * n + i) : 0.0f;
      else v = __ldg(ret + t * n + i);
    }
    tile[row][f] = v;
  }
  __syncthreads();
  const uint32_t rows = N - i0 < (uint32_t)kSmRows ? N - i0 : (uint32_t)kSmRows;
  float* out = dst + (t * n + i0) * Ws;
  for (int e = threadIdx.x; e < (int)rows * Ws; e += blockDim.x) {
    const int row = e / Ws, col = e - row * Ws;
    out[e] = col < F ? tile[row][col] : 0.0f;
  }
}

// k_gather from the sample-major copy: one row of Ws floats per sample, read
// in 16-byte pieces.
// Eight consecutive X values as 16-byte stores (X rows are multiples of 8
// elements, so every chunk starts on a 16-byte boundary).
__device__ __forceinline__ void st_act8(__nv_bfloat16* p, const float v[8]) {
  uint4 q;
  __nv_bfloat162 h0 = __floats2bfloat162_rn(v[0], v[1]), h1 = __floats2bfloat162_rn(v[2], v[3]);
  __nv_bfloat162 h2 = __floats2bfloat162_rn(v[4], v[5]), h3 = __floats2bfloat162_rn(v[6], v[7]);
  memcpy(&q.x, &h0, 4);
  memcpy(&q.y, &h1, 4);
  memcpy(&q.z, &h2, 4);
  memcpy(&q.w, &h3, 4);
  *reinterpret_cast<uint4*>(p) = q;
}
__device__ __forceinline__ void st_act8(float* p, const float v[8]) {
  reinterpret_cast<float4*>(p)[0] = make_float4(v[0], v[1], v[2], v[3]);
  reinterpret_cast<float4*>(p)[1] = make_float4(v[4], v[5], v[6], v[7]);
}

// A row of 8 words at p: one 256-bit access (a whole 32-byte L2 sector) when
// p is 32-byte aligned, else 16-byte pieces or single words.  A thread that
// writes its own sample's row otherwise covers a fraction of a sector per
// access, and the warp's 32 rows make 32 partial-sector requests.
__device__ __forceinline__ void st_row8(void* p, const uint32_t w[8]) {
  const uintptr_t a = reinterpret_cast<uintptr_t>(p);
  if (a % 32 == 0) {
    asm volatile("st.global.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(p), "r"(w[0]),
                 "r"(w[1]), "r"(w[2]), "r"(w[3]), "r"(w[4]), "r"(w[5]), "r"(w[6]), "r"(w[7])
                 : "memory");
  } else if (a % 16 == 0) {
    reinterpret_cast<uint4*>(p)[0] = make_uint4(w[0], w[1], w[2], w[3]);
    reinterpret_cast<uint4*>(p)[1] = make_uint4(w[4], w[5], w[6], w[7]);
  } else {
#pragma unroll
    for (int j = 0; j < 8; ++j) static_cast<uint32_t*>(p)[j] = w[j];
  }
}

__device__ __forceinline__ void ld_row8(const void* p, uint32_t w[8]) {
  const uintptr_t a = reinterpret_cast<uintptr_t>(p);
  if (a % 32 == 0) {
    asm volatile("ld.global.nc.v8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
                 : "=r"(w[0]), "=r"(w[1]), "=r"(w[2]), "=r"(w[3]), "=r"(w[4]), "=r"(w[5]),
                   "=r"(w[6]), "=r"(w[7])
                 : "l"(p));
  } else {
#pragma unroll
    for (int j = 0; j < 8; ++j) w[j] = __ldg(static_cast<const uint32_t*>(p) + j);
  }
}

// 2A head-gradient values of one sample (A = 8) as one row: bf16 pairs in
// one sector, or fp32 in two.
__device__ __forceinline__ void st_head16(__nv_bfloat16* p, const float v[16]) {
  uint32_t w[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(v[2 * j], v[2 * j + 1]);
    memcpy(&w[j], &h, 4);
  }
  st_row8(p, w);
}
__device__ __forceinline__ void st_head16(float* p, const float v[16]) {
  uint32_t w[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) w[j] = __float_as_uint(v[j]);
  st_row8(p, w);
#pragma unroll
  for (int j = 0; j < 8; ++j) w[j] = __float_as_uint(v[8 + j]);
  st_row8(p + 8, w);
}

// One sample per thread: its whole row (Ws <= W floats) is loaded at once
// and X is written in chunks of eight with vector stores; W is a
// compile-time bound on the row, so the row lives in registers.
template <typename TX, int W>
__global__ void __launch_bounds__(kT) k_gather_sm(Dims d, PermKey key, const StepCtl* ctl,
                                                  const float* __restrict__ rows, int Ws,
                                                  Sample out, TX* __restrict__ X) {
  __shared__ double sh[2 * (kT / 32)];
  const int b = blockIdx.x * kT + threadIdx.x;
  const unsigned long long epoch = ctl->epoch0 + ctl->step / ctl->n_mb;
  const uint32_t start = (ctl->step % ctl->n_mb) * (uint32_t)d.B;
  key.e0 = (uint32_t)epoch;
  key.e1 = (uint32_t)(epoch >> 32);
  double s[2] = {0.0, 0.0};
  if (b < d.B) {
    const uint32_t r = perm_index(start + (uint32_t)b, key);
    const float4* src = reinterpret_cast<const float4*>(rows + (size_t)r * Ws);
    float v[W];
#pragma unroll
    for (int q = 0; q < W / 4; ++q) {
      float4 t = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
      if (4 * q < Ws) t = __ldg(src + q);
      v[4 * q] = t.x;
      v[4 * q + 1] = t.y;
      v[4 * q + 2] = t.z;
      v[4 * q + 3] = t.w;
    }
    TX* x = X + (size_t)b * d.Dp;
#pragma unroll
    for (int c = 0; c < W / 8; ++c) {
      if (8 * c < d.Dp) {
        float x8[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const int k = 8 * c + j;
          x8[j] = k < d.D ? v[k] : (k == d.D ? 1.0f : 0.0f);
        }
        st_act8(x + 8 * c, x8);
      }
    }
    // the fields after the observation sit at run-time offsets: read them
    // from the row again (its sectors are in L1 from the loads above), so
    // that v stays in registers
    const float* f = rows + (size_t)r * Ws + d.D;
    if (!d.value_only && d.A == 8) {
      uint32_t w[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) w[j] = __float_as_uint(__ldg(f + j));
      st_row8(out.act + (size_t)b * 8, w);
    } else if (!d.value_only) {
      for (int j = 0; j < d.A; ++j) out.act[(size_t)b * d.A + j] = __ldg(f + j);
    }
    const float lp = __ldg(f + d.A), a = __ldg(f + d.A + 1);
    out.ret[b] = __ldg(f + d.A + 2);
    if (!d.value_only) {
      out.logp[b] = lp;
      out.adv[b] = a;
      s[0] = a;
      s[1] = (double)a * a;
    }
  }
  block_sum<2>(s, sh);
  if (threadIdx.x == 0) {
    out.adv_part[2 * blockIdx.x] = s[0];
    out.adv_part[2 * blockIdx.x + 1] = s[1];
  }
}

__global__ void __launch_bounds__(kT) k_tanh_fwd(float* __restrict__ h, int ld, int B, int H4) {
  const size_t n = (size_t)B * H4;
  for (size_t e = blockIdx.x * (size_t)kT + threadIdx.x; e < n; e += (size_t)gridDim.x * kT) {
    const size_t row = e / H4, c = e - row * H4;
    float4* p = reinterpret_cast<float4*>(h + row * ld) + c;
    float4 z = *p;
    z.x = tanhf(z.x); z.y = tanhf(z.y); z.z = tanhf(z.z); z.w = tanhf(z.w);
    *p = z;
  }
}

__global__ void __launch_bounds__(kT) k_tanh_fwd_bf16(__nv_bfloat16* __restrict__ h, int ld,
                                                      int B, int H8) {
  const size_t n = (size_t)B * H8;
  for (size_t e = blockIdx.x * (size_t)kT + threadIdx.x; e < n; e += (size_t)gridDim.x * kT) {
    const size_t row = e / H8, c = e - row * H8;
    uint4* p = reinterpret_cast<uint4*>(h + row * ld) + c;
    uint4 u = *p;
    __nv_bfloat162* v = reinterpret_cast<__nv_bfloat162*>(&u);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const float2 z = __bfloat1622float2(v[k]);
      v[k] = __floats2bfloat162_rn(tanhf(z.x), tanhf(z.y));
    }
    *p = u;
  }
}

__global__ void __launch_bounds__(kT) k_tanh_bwd_bf16(__nv_bfloat16* __restrict__ g, int ldg,
                                                      const __nv_bfloat16* __restrict__ h,
                                                      int ldh, int B, int H8) {
  const size_t n = (size_t)B * H8;
  for (size_t e = blockIdx.x * (size_t)kT + threadIdx.x; e < n; e += (size_t)gridDim.x * kT) {
    const size_t row = e / H8, c = e - row * H8;
    uint4* pg = reinterpret_cast<uint4*>(g + row * ldg) + c;
    uint4 hv = __ldg(reinterpret_cast<const uint4*>(h + row * ldh) + c);
    uint4 gv = *pg;
    __nv_bfloat162* gg = reinterpret_cast<__nv_bfloat162*>(&gv);
    const __nv_bfloat162* hh = reinterpret_cast<const __nv_bfloat162*>(&hv);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const float2 y = __bfloat1622float2(hh[k]);
      const float2 x = __bfloat1622float2(gg[k]);
      gg[k] = __floats2bfloat162_rn(x.x * (1.0f - y.x * y.x), x.y * (1.0f - y.y * y.y));
    }
    *pg = gv;
  }
}

__global__ void __launch_bounds__(kT) k_tanh_bwd(float* __restrict__ g, int ldg,
                                                 const float* __restrict__ h, int ldh, int B,
                                                 int H4) {
  const size_t n = (size_t)B * H4;
  for (size_t e = blockIdx.x * (size_t)kT + threadIdx.x; e < n; e += (size_t)gridDim.x * kT) {
    const size_t row = e / H4, c = e - row * H4;
    float4* pg = reinterpret_cast<float4*>(g + row * ldg) + c;
    const float4 y = __ldg(reinterpret_cast<const float4*>(h + row * ldh) + c);
    float4 v = *pg;
    v.x *= 1.0f - y.x * y.x; v.y *= 1.0f - y.y * y.y;
    v.z *= 1.0f - y.z * y.z; v.w *= 1.0f - y.w * y.w;
    *pg = v;
  }
}

// One thread per sample: log-density, ratio, clipped surrogate, value and
// entropy terms, and dL/d(head) for both networks (already divided by B).
// Every block first reduces the gather's advantage partial sums, in the same
// order, so that all blocks normalise with the same mean and deviation.
template <typename TG>
__global__ void __launch_bounds__(kT) k_head(Dims d, LossHp hp, const float* __restrict__ y,
                                             const float* __restrict__ v, Sample smp,
                                             int n_part, TG* __restrict__ g_y,
                                             TG* __restrict__ g_v, float* __restrict__ part) {
  __shared__ double shd[2 * (kT / 32)];
  __shared__ float shf[5 * (kT / 32)];
  __shared__ double norm[2];
  double s[2] = {0.0, 0.0};
  for (int k = threadIdx.x; k < n_part; k += kT) {
    s[0] += smp.adv_part[2 * k];
    s[1] += smp.adv_part[2 * k + 1];
  }
  block_sum<2>(s, shd);
  if (threadIdx.x == 0) {
    const double mean = s[0] / d.B;
    const double var = fmax((s[1] - s[0] * mean) / (d.B - 1), 0.0);
    norm[0] = mean;
    norm[1] = 1.0 / (sqrt(var) + 1e-8);
  }
  __syncthreads();
  const int b = blockIdx.x * kT + threadIdx.x;
  float st[5] = {0.f, 0.f, 0.f, 0.f, 0.f};
  if (b < d.B && d.value_only) {
    const float dv = v[(size_t)b * d.ld_val] - smp.ret[b];
    st_act(g_v + (size_t)b * d.ld_val, hp.vf_coef * dv * (1.0f / (float)d.B));
    st[1] = 0.5f * dv * dv;
  } else if (b < d.B) {
    const float inv_b = 1.0f / (float)d.B;
    const int A = d.A;
    const float* yb = y + (size_t)b * d.ld_pol;
    const float* ab = smp.act + (size_t)b * A;
    const float an = hp.norm_adv ? (float)(((double)smp.adv[b] - norm[0]) * norm[1]) : smp.adv[b];
    float dm[8], iv[8], z2[8];
    bool in[8];
    float lp = -(float)A * kHalfLog2Pi, ent = (float)A * (0.5f + kHalfLog2Pi);
    // A = 8: the sample's 16 head outputs and 8 actions as whole sectors
    float yv[16], av[8];
    if (A == 8) {
      uint32_t w[8];
      ld_row8(yb, w);
#pragma unroll
      for (int j = 0; j < 8; ++j) yv[j] = __uint_as_float(w[j]);
      ld_row8(yb + 8, w);
#pragma unroll
      for (int j = 0; j < 8; ++j) yv[8 + j] = __uint_as_float(w[j]);
      ld_row8(ab, w);
#pragma unroll
      for (int j = 0; j < 8; ++j) av[j] = __uint_as_float(w[j]);
    }
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      if (k < A) {
        const float raw = A == 8 ? yv[8 + k] : yb[A + k];
        const float ls = fminf(fmaxf(raw, hp.logstd_min), hp.logstd_max);
        in[k] = raw >= hp.logstd_min && raw <= hp.logstd_max;
        iv[k] = expf(-2.0f * ls);
        dm[k] = A == 8 ? av[k] - yv[k] : ab[k] - yb[k];
        z2[k] = dm[k] * dm[k] * iv[k];
        lp += -0.5f * z2[k] - ls;
        ent += ls;
      }
    }
    const float lp_old = smp.logp[b];
    const float r = expf(lp - lp_old);
    const float lo = 1.0f - hp.clip_eps, hi = 1.0f + hp.clip_eps;
    const bool unclipped = an > 0.0f ? r <= hi : r >= lo;
    const float g_lp = unclipped ? -an * r * inv_b : 0.0f;
    TG* gy = g_y + (size_t)b * d.ld_pol;
    if (A == 8) {
      float gv[16];
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        gv[k] = g_lp * dm[k] * iv[k];
        gv[8 + k] = in[k] ? g_lp * (z2[k] - 1.0f) - hp.ent_coef * inv_b : 0.0f;
      }
      st_head16(gy, gv);
    } else {
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        if (k < A) {
          st_act(gy + k, g_lp * dm[k] * iv[k]);
          st_act(gy + A + k, in[k] ? g_lp * (z2[k] - 1.0f) - hp.ent_coef * inv_b : 0.0f);
        }
      }
    }
    const float dv = v[(size_t)b * d.ld_val] - smp.ret[b];
    st_act(g_v + (size_t)b * d.ld_val, hp.vf_coef * dv * inv_b);
    st[0] = fmaxf(-an * r, -an * fminf(fmaxf(r, lo), hi));
    st[1] = 0.5f * dv * dv;
    st[2] = ent;
    st[3] = lp_old - lp;
    st[4] = fabsf(r - 1.0f) > hp.clip_eps ? 1.0f : 0.0f;
  }
  block_sum<5>(st, shf);
  if (threadIdx.x == 0)
    for (int k = 0; k < 5; ++k) part[5 * blockIdx.x + k] = st[k];
}

__global__ void __launch_bounds__(kT) k_stats(int B, int n_part, float vf_coef, float ent_coef,
                                              const float* __restrict__ part, float* mb,
                                              float* acc) {
  // (value-only steps leave the policy terms of part at 0).  fp32 sums of the
  // per-block fp32 partials: the GPU's fp64 pipe made this one-block kernel
  // take about 10 us, for statistics that are reported, not trained on.
  __shared__ float sh[5 * (kT / 32)];
  float s[5] = {0, 0, 0, 0, 0};
  for (int k = threadIdx.x; k < n_part; k += kT)
    for (int j = 0; j < 5; ++j) s[j] += part[5 * k + j];
  block_sum<5>(s, sh);
  if (threadIdx.x == 0) {
    float r[8];
    const float inv_b = 1.0f / (float)B;
    for (int j = 0; j < 5; ++j) r[j] = s[j] * inv_b;
    r[5] = 0.0f;
    r[6] = r[0] + vf_coef * r[1] - ent_coef * r[2];
    r[7] = 1.0f;
    for (int j = 0; j < 8; ++j) mb[j] = r[j];
    if (acc)
      for (int j = 0; j < 8; ++j)
        if (j != 5) acc[j] += r[j];
  }
}

__global__ void __launch_bounds__(kT) k_sumsq(const float* __restrict__ g, size_t n,
                                              float* __restrict__ part) {
  __shared__ float sh[kT / 32];
  float s[1] = {0.0f};
  for (size_t e = blockIdx.x * (size_t)kT + threadIdx.x; e < n; e += (size_t)gridDim.x * kT) {
    const float x = g[e];
    s[0] = fmaf(x, x, s[0]);
  }
  block_sum<1>(s, sh);
  if (threadIdx.x == 0) part[blockIdx.x] = s[0];
}

// The clip scale of the global gradient norm and the bias corrections of
// step t + 1, once per step (one block; the partials summed in index order):
// part[kNormBlocks + 0, 1, 2] = scale, 1 - b1^(t+1), 1 - b2^(t+1).
__global__ void __launch_bounds__(kT) k_adam_prep(float* __restrict__ part, AdamHp hp,
                                                  const StepCtl* ctl, float* mb, float* acc) {
  __shared__ float sh[kT / 32];
  float s[1] = {0.0f};
  for (int k = threadIdx.x; k < kNormBlocks; k += kT) s[0] += part[k];
  block_sum<1>(s, sh);
  if (threadIdx.x == 0) {
    // fp32 throughout: on the GPU's fp64 pipe a double pow takes microseconds
    const float norm = sqrtf(s[0]);
    part[kNormBlocks] = hp.max_norm > 0.0f ? fminf(1.0f, hp.max_norm / (norm + 1e-6f)) : 1.0f;
    // 1 - b^t as -expm1(t log b); b = 0 keeps the plain moment
    const float t1 = (float)(ctl->t + 1ull);
    const float c1 = hp.b1 > 0.0f ? -expm1f(t1 * logf(hp.b1)) : 1.0f;
    const float c2 = hp.b2 > 0.0f ? -expm1f(t1 * logf(hp.b2)) : 1.0f;
    part[kNormBlocks + 1] = c1 > 0.0f ? c1 : 1.0f;
    part[kNormBlocks + 2] = c2 > 0.0f ? c2 : 1.0f;
    mb[5] = norm;
    if (acc) acc[5] += norm;
  }
}

// One Adam step on the clipped gradient (scalars from k_adam_prep).
__global__ void __launch_bounds__(kT) k_adam(float* __restrict__ w, const float* __restrict__ g,
                                             float* __restrict__ m, float* __restrict__ v,
                                             size_t n, const float* __restrict__ part, AdamHp hp,
                                             __nv_bfloat16* __restrict__ wb) {
  const float scale = part[kNormBlocks];
  const float c1 = part[kNormBlocks + 1], c2 = part[kNormBlocks + 2];
  const float ib1 = 1.0f - hp.b1, ib2 = 1.0f - hp.b2;
  for (size_t e = blockIdx.x * (size_t)kT + threadIdx.x; e < n; e += (size_t)gridDim.x * kT) {
    const float gi = g[e] * scale;
    const float mi = hp.b1 * m[e] + ib1 * gi;
    const float vi = hp.b2 * v[e] + ib2 * gi * gi;
    m[e] = mi;
    v[e] = vi;
    const float wi = w[e] - hp.lr * (mi / c1) / (sqrtf(vi / c2) + hp.eps);
    w[e] = wi;
    if (wb) wb[e] = __float2bfloat16_rn(wi);
  }
}

__global__ void __launch_bounds__(kT) k_to_bf16(const float* __restrict__ w,
                                                __nv_bfloat16* __restrict__ wb, size_t n) {
  for (size_t e = blockIdx.x * (size_t)kT + threadIdx.x; e < n; e += (size_t)gridDim.x * kT)
    wb[e] = __float2bfloat16_rn(w[e]);
}

__global__ void k_step_advance(StepCtl* ctl) {
  ctl->step += 1u;
  ctl->t += 1ull;
}

__global__ void k_finish(const float* __restrict__ acc, float* __restrict__ out) {
  const int j = threadIdx.x;
  if (j < 8) {
    const float steps = acc[7];
    out[j] = j == 7 ? steps : acc[j] / steps;
  }
}

// Flat index of augmented element e (-1 for a padding element).
__device__ __forceinline__ long long flat_index(size_t e, int in, int in_p, int H, int Hp,
                                                int out) {
  const size_t n1 = (size_t)H * in_p, n2 = (size_t)H * Hp;
  const long long b1 = (long long)H * in, w2 = b1 + H, b2 = w2 + (long long)H * H,
                  w3 = b2 + H, b3 = w3 + (long long)out * H;
  if (e < n1) {
    const int row = (int)(e / in_p), col = (int)(e - (size_t)row * in_p);
    return col < in ? (long long)row * in + col : col == in ? b1 + row : -1;
  }
  e -= n1;
  if (e < n2) {
    const int row = (int)(e / Hp), col = (int)(e - (size_t)row * Hp);
    return col < H ? w2 + (long long)row * H + col : col == H ? b2 + row : -1;
  }
  e -= n2;
  const int row = (int)(e / Hp), col = (int)(e - (size_t)row * Hp);
  return col < H ? w3 + (long long)row * H + col : col == H ? b3 + row : -1;
}

__device__ void convert_range(float* flat, float* aug, size_t n_aug, int in, int in_p, int H, int Hp,
                              int out, int to_aug) {
  for (size_t e = blockIdx.x * (size_t)kT + threadIdx.x; e < n_aug; e += (size_t)gridDim.x * kT) {
    const long long f = flat_index(e, in, in_p, H, Hp, out);
    if (to_aug)
      aug[e] = f >= 0 ? flat[f] : 0.0f;
    else if (f >= 0)
      flat[f] = aug[e];
  }
}

__global__ void __launch_bounds__(kT) k_convert(float* flat, float* aug, size_t n_aug, int in,
                                                int in_p, int H, int Hp, int out, int to_aug) {
  convert_range(flat, aug, n_aug, in, in_p, H, Hp, out, to_aug);
}

// Both networks in one launch: blockIdx.y = 0 policy, 1 value.
struct ConvertPair {
  float* flat[2];
  float* aug[2];
  int out[2];
  size_t n_aug[2];
};
__global__ void __launch_bounds__(kT) k_convert_pair(const ConvertPair c, int in, int in_p, int H,
                                                     int Hp, int to_aug) {
  const int net = blockIdx.y;
  convert_range(c.flat[net], c.aug[net], c.n_aug[net], in, in_p, H, Hp, c.out[net], to_aug);
}

template <typename TX>
__global__ void __launch_bounds__(kT) k_fill_ones(TX* buf, int ld, int col, int rows) {
  for (int r = blockIdx.x * kT + threadIdx.x; r < rows; r += gridDim.x * kT) {
    TX* p = buf + (size_t)r * ld;
    st_act(p + col, 1.0f);
    for (int c = col + 1; c < ld; ++c) st_act(p + c, 0.0f);
  }
}

unsigned grid_for(size_t n) {
  const size_t g = (n + kT - 1) / kT;
  return (unsigned)(g < 152 * 8 ? (g > 0 ? g : 1) : 152 * 8);
}

}  // namespace

size_t aug_count(int in, int in_p, int H, int Hp, int out) {
  return (size_t)H * in_p + (size_t)H * Hp + (size_t)out * Hp;
}

cudaError_t launch_gather(const Dims& d, const PermKey& k, const StepCtl* ctl, const float* obs,
                          const float* act, const float* logp, const float* adv,
                          const float* ret, uint32_t N, const Sample& out, void* X,
                          cudaStream_t s) {
  const unsigned nb = (d.B + kT - 1) / kT;
  if (d.bf16)
    k_gather<<<nb, kT, 0, s>>>(d, k, ctl, obs, act, logp, adv, ret, N, out,
                               static_cast<__nv_bfloat16*>(X));
  else
    k_gather<<<nb, kT, 0, s>>>(d, k, ctl, obs, act, logp, adv, ret, N, out,
                               static_cast<float*>(X));
  return cudaGetLastError();
}

int sample_row_floats(int D, int A) { return (D + A + 3 + 7) & ~7; }

cudaError_t launch_transpose_batch(int D, int A, uint32_t T, uint32_t N, const float* obs,
                                   const float* act, const float* logp, const float* adv,
                                   const float* ret, float* dst, cudaStream_t s) {
  const int Ws = sample_row_floats(D, A);
  if (Ws > kSmMaxW) return cudaErrorInvalidValue;
  const size_t blocks = (size_t)T * ((N + kSmRows - 1) / kSmRows);
  if (blocks == 0 || blocks > 0x7fffffffu) return cudaErrorInvalidValue;
  k_transpose_batch<<<(unsigned)blocks, 256, 0, s>>>(D, A, Ws, N, obs, act, logp, adv, ret, dst);
  return cudaGetLastError();
}

cudaError_t launch_gather_sm(const Dims& d, const PermKey& k, const StepCtl* ctl,
                             const float* rows, const Sample& out, void* X, cudaStream_t s) {
  const unsigned nb = (d.B + kT - 1) / kT;
  const int Ws = sample_row_floats(d.D, d.A);
  if (Ws > kSmMaxW || d.Dp > Ws || d.Dp % 8 != 0 || reinterpret_cast<uintptr_t>(X) % 16 != 0 ||
      reinterpret_cast<uintptr_t>(rows) % 16 != 0)
    return cudaErrorInvalidValue;
  if (d.bf16) {
    __nv_bfloat16* xb = static_cast<__nv_bfloat16*>(X);
    if (Ws <= 32) k_gather_sm<__nv_bfloat16, 32><<<nb, kT, 0, s>>>(d, k, ctl, rows, Ws, out, xb);
    else k_gather_sm<__nv_bfloat16, kSmMaxW><<<nb, kT, 0, s>>>(d, k, ctl, rows, Ws, out, xb);
  } else {
    float* xf = static_cast<float*>(X);
    if (Ws <= 32) k_gather_sm<float, 32><<<nb, kT, 0, s>>>(d, k, ctl, rows, Ws, out, xf);
    else k_gather_sm<float, kSmMaxW><<<nb, kT, 0, s>>>(d, k, ctl, rows, Ws, out, xf);
  }
  return cudaGetLastError();
}

cudaError_t launch_step_advance(StepCtl* ctl, cudaStream_t s) {
  k_step_advance<<<1, 1, 0, s>>>(ctl);
  return cudaGetLastError();
}

cudaError_t launch_tanh_fwd(bool bf16, void* h, int ld, int B, int H, cudaStream_t s) {
  if (bf16)
    k_tanh_fwd_bf16<<<grid_for((size_t)B * H / 8), kT, 0, s>>>(static_cast<__nv_bfloat16*>(h), ld,
                                                               B, H / 8);
  else
    k_tanh_fwd<<<grid_for((size_t)B * H / 4), kT, 0, s>>>(static_cast<float*>(h), ld, B, H / 4);
  return cudaGetLastError();
}

cudaError_t launch_tanh_bwd(bool bf16, void* g, int ldg, const void* h, int ldh, int B, int H,
                            cudaStream_t s) {
  if (bf16)
    k_tanh_bwd_bf16<<<grid_for((size_t)B * H / 8), kT, 0, s>>>(
        static_cast<__nv_bfloat16*>(g), ldg, static_cast<const __nv_bfloat16*>(h), ldh, B, H / 8);
  else
    k_tanh_bwd<<<grid_for((size_t)B * H / 4), kT, 0, s>>>(static_cast<float*>(g), ldg,
                                                          static_cast<const float*>(h), ldh, B,
                                                          H / 4);
  return cudaGetLastError();
}

cudaError_t launch_head(const Dims& d, const LossHp& hp, const float* y, const float* v,
                        const Sample& smp, void* g_y, void* g_v, float* part, cudaStream_t s) {
  const int nb = (d.B + kT - 1) / kT;
  if (d.bf16)
    k_head<<<nb, kT, 0, s>>>(d, hp, y, v, smp, nb, static_cast<__nv_bfloat16*>(g_y),
                             static_cast<__nv_bfloat16*>(g_v), part);
  else
    k_head<<<nb, kT, 0, s>>>(d, hp, y, v, smp, nb, static_cast<float*>(g_y),
                             static_cast<float*>(g_v), part);
  return cudaGetLastError();
}

cudaError_t launch_stats(const Dims& d, const LossHp& hp, const float* part, float* mb,
                         float* acc, cudaStream_t s) {
  k_stats<<<1, kT, 0, s>>>(d.B, (d.B + kT - 1) / kT, hp.vf_coef, hp.ent_coef, part, mb, acc);
  return cudaGetLastError();
}

cudaError_t launch_adam(float* w, const float* g, float* m, float* v, size_t n, float* part,
                        const AdamHp& hp, const StepCtl* ctl, float* mb, float* acc, void* wb,
                        cudaStream_t s) {
  k_sumsq<<<kNormBlocks, kT, 0, s>>>(g, n, part);
  k_adam_prep<<<1, kT, 0, s>>>(part, hp, ctl, mb, acc);
  k_adam<<<grid_for(n), kT, 0, s>>>(w, g, m, v, n, part, hp, static_cast<__nv_bfloat16*>(wb));
  return cudaGetLastError();
}

cudaError_t launch_to_bf16(const float* w, void* wb, size_t n, cudaStream_t s) {
  k_to_bf16<<<grid_for(n), kT, 0, s>>>(w, static_cast<__nv_bfloat16*>(wb), n);
  return cudaGetLastError();
}

cudaError_t launch_finish(const float* acc, float* out, cudaStream_t s) {
  k_finish<<<1, 32, 0, s>>>(acc, out);
  return cudaGetLastError();
}

cudaError_t launch_convert(float* flat, float* aug, int in, int in_p, int H, int Hp, int out,
                           bool to_aug, cudaStream_t s) {
  const size_t n = aug_count(in, in_p, H, Hp, out);
  k_convert<<<grid_for(n), kT, 0, s>>>(flat, aug, n, in, in_p, H, Hp, out, to_aug ? 1 : 0);
  return cudaGetLastError();
}

cudaError_t launch_convert_pair(float* flat_pol, float* aug_pol, int out_pol, float* flat_val,
                                float* aug_val, int out_val, int in, int in_p, int H, int Hp,
                                bool to_aug, cudaStream_t s) {
  const ConvertPair c = {{flat_pol, flat_val},
                         {aug_pol, aug_val},
                         {out_pol, out_val},
                         {aug_count(in, in_p, H, Hp, out_pol), aug_count(in, in_p, H, Hp, out_val)}};
  const size_t n = c.n_aug[0] > c.n_aug[1] ? c.n_aug[0] : c.n_aug[1];
  k_convert_pair<<<dim3(grid_for(n), 2), kT, 0, s>>>(c, in, in_p, H, Hp, to_aug ? 1 : 0);
  return cudaGetLastError();
}

cudaError_t launch_fill_ones(bool bf16, void* buf, int ld, int col, int rows, cudaStream_t s) {
  if (bf16)
    k_fill_ones<<<grid_for((size_t)rows), kT, 0, s>>>(static_cast<__nv_bfloat16*>(buf), ld, col,
                                                      rows);
  else
    k_fill_ones<<<grid_for((size_t)rows), kT, 0, s>>>(static_cast<float*>(buf), ld, col, rows);
  return cudaGetLastError();
}

}  // namespace ppo
}  // namespace auv
