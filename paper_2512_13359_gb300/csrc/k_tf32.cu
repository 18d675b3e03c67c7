// k_tf32.cu -- the fused rollout with fp32 networks on the tensor cores
// (tcgen05 kind::tf32): the 18 -> 256 -> 256 -> 8 (or 16) policy of the
// fp32 workloads, whose layers run with tf32 operands (weights, inputs and
// hidden activations rounded to nearest tf32) and fp32 accumulation, biases
// and tanh in fp32.
//
// One CTA per tile of 128 envs (one thread per env; its row of every tile is
// its tensor-memory lane), one MMA-issuing warp and one producer warp.  Per
// control step:
//   observation -> obs tile (smem, 32 fp32 columns, 18 used)
//   layer 1: D[0, 256) = obs x W1^T          (W1 resident in smem)
//   epilogue: + b1, tanh, round to tf32, written back in place (tcgen05.st),
//            32 columns at a time, each chunk announced as soon as it is in
//            tensor memory
//   layer 2: D[256, 512) = h1 (A from tensor memory) x W2^T, K-slice j
//            issued once h1's chunk j is written (so it runs while the
//            epilogue computes the later chunks), W2 streamed
//            through a four-stage ring of 32 KB K-slices by bulk copies
//            (256 KB of fp32 W2 does not fit beside the rest; the producer
//            runs ahead, so the next step's first slices load during the
//            current step's physics)
//   epilogue: + b2, tanh, tf32, in place, each 32-column chunk announced
//   layer 3: D[0, 16) = h2 (tensor memory) x W3^T (resident), K-slice j
//            issued once h2's chunk j is written (layer 2 has completed, so
//            h1's columns are free for its accumulator)
//   head: + b3 -> Gaussian action, physics substeps, reward, done, reset
// Every wait is an mbarrier wait bounded by 2 s; a timeout raises the CTA's
// abort flag and latches AUV_ERR_TIMEOUT in the status block.
#include "auv_kernels.h"
#include "auv_bf16.h"
#include "tc_ptx.cuh"

namespace auv {
namespace {

constexpr int kH = 256;
constexpr int kRows = 128;
constexpr int kSlices = 8;                        // W2 K-slices of 32 fp32
constexpr uint32_t kSliceBytes = kH * 128;        // 256 rows x 128 B
constexpr int kRing = 4;
constexpr uint64_t kWaitLimitNs = 2000000000ull;

// Packed image (global memory), 128-byte-swizzled K-major operand tiles:
// W1 [256 rows x 32 K], W2 as 8 K-slices [256 x 32], W3 as 8 K-slices
// [16 x 32] (rows past the head width zero), then fp32 b1[256], b2[256],
// b3[16].  Weights rounded to tf32 (nearest, ties away).
constexpr uint32_t kOffW1 = 0;
constexpr uint32_t kOffW2 = kOffW1 + kH * 128;
constexpr uint32_t kOffW3 = kOffW2 + kSlices * kSliceBytes;
constexpr uint32_t kW3Slice = 16 * 128;
constexpr uint32_t kOffB = kOffW3 + kSlices * kW3Slice;
constexpr uint32_t kImage = kOffB + (2 * kH + 16) * 4;

// Shared memory: W1 | W3 | biases | obs tile | W2 ring | barriers.
constexpr uint32_t kSW1 = 0;
constexpr uint32_t kSW3 = kSW1 + kH * 128;
constexpr uint32_t kSB = kSW3 + kSlices * kW3Slice;
constexpr uint32_t kSObs = (kSB + (2 * kH + 16) * 4 + 1023) & ~1023u;
constexpr uint32_t kSRing = kSObs + kRows * 128;
constexpr uint32_t kSBar = kSRing + kRing * kSliceBytes;

struct Bars {
  uint64_t img_full, obs_full, l1_full, l2_full, l3_full, drain;
  uint64_t h1_part[kSlices];   // h1 columns 32j..32j+31 written (128 arrivals): layer-2 K-slice j may run
  uint64_t h2_part[kSlices];   // h2 columns 256+32j.. written (128 arrivals): layer-3 K-slice j may run
  uint64_t w2_full[kRing], w2_empty[kRing];
  uint32_t tmem_base;
  int abort;
};
constexpr uint32_t kSmem = kSBar + sizeof(Bars) + 1024;

__device__ __forceinline__ float to_tf32(float x) {
  uint32_t r;
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
  return __uint_as_float(r);
}

// Element (n, k) of a 128-byte-swizzled K-major tile of 32 fp32 per row.
__device__ __forceinline__ uint32_t sw_off(int n, int k) {
  return (uint32_t)n * 128 + ((uint32_t)((k >> 2) ^ (n & 7)) << 4) + (uint32_t)(k & 3) * 4;
}

__global__ void k_pack_tf32(const float* __restrict__ w, int in_dim, int out_dim,
                            uint8_t* __restrict__ img) {
  const float* W1 = w;
  const float* b1 = W1 + kH * in_dim;
  const float* W2 = b1 + kH;
  const float* b2 = W2 + kH * kH;
  const float* W3 = b2 + kH;
  const float* b3 = W3 + out_dim * kH;
  const int id = blockIdx.x * blockDim.x + threadIdx.x;
  const int n1 = kH * 32, n2 = kH * kH, n3 = kSlices * 16 * 32;
  if (id < n1) {
    const int n = id >> 5, k = id & 31;
    const float v = k < in_dim ? to_tf32(W1[n * in_dim + k]) : 0.0f;
    *reinterpret_cast<float*>(img + kOffW1 + sw_off(n, k)) = v;
  } else if (id < n1 + n2) {
    const int e = id - n1, n = e / kH, k = e % kH;
    *reinterpret_cast<float*>(img + kOffW2 + (k >> 5) * kSliceBytes + sw_off(n, k & 31)) =
        to_tf32(W2[n * kH + k]);
  } else if (id < n1 + n2 + n3) {
    const int e = id - n1 - n2, j = e / (16 * 32), n = (e / 32) % 16, k = e % 32;
    const float v = n < out_dim ? to_tf32(W3[n * kH + 32 * j + k]) : 0.0f;
    *reinterpret_cast<float*>(img + kOffW3 + j * kW3Slice + sw_off(n, k)) = v;
  } else {
    const int e = id - n1 - n2 - n3;
    float* f = reinterpret_cast<float*>(img + kOffB);
    if (e < kH) f[e] = b1[e];
    else if (e < 2 * kH) f[e] = b2[e - kH];
    else if (e < 2 * kH + 16) f[e] = e - 2 * kH < out_dim ? b3[e - 2 * kH] : 0.0f;
  }
}

// Shared-memory descriptor of a 128-byte-swizzled K-major tile (8-row groups
// 1024 bytes apart).
__device__ __forceinline__ uint64_t desc(uint32_t saddr) {
  return tc::smem_desc(saddr, 1024, 2);
}

// kind::tf32 instruction descriptor: D fp32, A and B tf32, K-major, M x N.
__host__ __device__ constexpr uint32_t idesc_tf32(int M, int N) {
  return (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(N >> 3) << 17) |
         ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void mma_ss(uint32_t d, uint64_t a, uint64_t b, uint32_t id,
                                       uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}" ::"r"(d),
      "l"(a), "l"(b), "r"(id), "r"(acc)
      : "memory");
}

__device__ __forceinline__ void mma_ts(uint32_t d, uint32_t a_tmem, uint64_t b, uint32_t id,
                                       uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::tf32 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d),
      "r"(a_tmem), "l"(b), "r"(id), "r"(acc)
      : "memory");
}

__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, "
      "%17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(
          taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
      "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]),
      "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]),
      "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}

// Hidden layer epilogue for this thread's row: 256 accumulator columns at
// col0 -> + bias -> tanh -> tf32, written back in place.  With `part` set,
// each 32-column chunk is announced as soon as it is in tensor memory
// (part[c], one arrival per thread), so that the next layer's K-slice c can
// start while the later chunks are still being computed.
__device__ __forceinline__ void hidden_epilogue(uint32_t lane_addr, uint32_t col0,
                                                const float* bias, uint64_t* part = nullptr) {
#pragma unroll 1
  for (int c = 0; c < kH / 32; ++c) {
    uint32_t acc[32];
    tc::tmem_ld32(lane_addr + col0 + 32 * c, acc);
    tc::tmem_ld_wait(acc);
#pragma unroll
    for (int j = 0; j < 32; ++j)
      acc[j] = __float_as_uint(
          to_tf32(tc::tanh_f32(__uint_as_float(acc[j]) + bias[32 * c + j])));
    tmem_st32(lane_addr + col0 + 32 * c, acc);
    if (part) {
      tc::tmem_st_wait();
      tc::tc_fence_before();
      tc::mbar_arrive(&part[c]);
    }
  }
  tc::tmem_st_wait();
}

// Gaussian head and the step's normals -> action and log-density (the fp32
// path's sampling: the accurate log, sine and exponential).
__device__ __forceinline__ void sample(const Model& M, const float* head, const float eps[kAct],
                                       float a[kAct], float* logp) {
  float lp = 0.0f;
#pragma unroll
  for (int k = 0; k < kAct; ++k) {
    float ls = M.logstd_fixed[k];
    if (M.policy_out == 16) ls = fminf(fmaxf(head[kAct + k], M.logstd_min), M.logstd_max);
    a[k] = fmaf(expf(ls), eps[k], head[k]);
    lp += -0.5f * eps[k] * eps[k] - ls;
  }
  *logp = lp - (float)kAct * 0.91893853320467274f;
}

__global__ void __launch_bounds__(192, 1)
k_rollout_tf32(const Model M, Buffers B, const uint8_t* __restrict__ image, Traj tr, int T,
               uint64_t t_g0, Status* st) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023u) & ~(uintptr_t)1023u);
  Bars* bar = reinterpret_cast<Bars*>(smem + kSBar);
  volatile int* abort = &bar->abort;
  const int tid = threadIdx.x, warp = tid >> 5;

  if (tid == 0) {
    tc::mbar_init(&bar->img_full, 1);
    tc::mbar_init(&bar->obs_full, kRows);
    tc::mbar_init(&bar->l1_full, 1);
    for (int j = 0; j < kSlices; ++j) tc::mbar_init(&bar->h1_part[j], kRows);
    tc::mbar_init(&bar->l2_full, 1);
    for (int j = 0; j < kSlices; ++j) tc::mbar_init(&bar->h2_part[j], kRows);
    tc::mbar_init(&bar->l3_full, 1);
    tc::mbar_init(&bar->drain, 1);
    for (int s = 0; s < kRing; ++s) {
      tc::mbar_init(&bar->w2_full[s], 1);
      tc::mbar_init(&bar->w2_empty[s], 1);
    }
    bar->abort = 0;
    tc::mbar_fence_init();
    // resident pieces: W1, W3 and the biases
    tc::mbar_arrive_expect_tx(&bar->img_full, kH * 128 + kSlices * kW3Slice + (2 * kH + 16) * 4);
    tc::bulk_g2s(smem + kSW1, image + kOffW1, kH * 128, &bar->img_full);
    tc::bulk_g2s(smem + kSW3, image + kOffW3, kSlices * kW3Slice, &bar->img_full);
    tc::bulk_g2s(smem + kSB, image + kOffB, (2 * kH + 16) * 4, &bar->img_full);
  }
  if (warp == 4) {
    tc::tmem_alloc(&bar->tmem_base, 512);
    tc::tmem_relinquish();
  }
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = bar->tmem_base;
  const uint32_t s_base = tc::smem_u32(smem);
  const bool img_ok = tc::mbar_wait(&bar->img_full, 0, abort, kWaitLimitNs);
  const int steps = img_ok ? T : 0;

  if (warp == 5) {
    // ---- producer: W2 K-slices into the ring, 8 per control step ----
    if ((tid & 31) == 0) {
      const int total = steps * kSlices;
      for (int g = 0; g < total; ++g) {
        const int s = g % kRing;
        if (g >= kRing &&
            !tc::mbar_wait(&bar->w2_empty[s], (uint32_t)(g / kRing - 1) & 1u, abort, kWaitLimitNs))
          break;
        tc::mbar_arrive_expect_tx(&bar->w2_full[s], kSliceBytes);
        tc::bulk_g2s(smem + kSRing + s * kSliceBytes, image + kOffW2 + (g % kSlices) * kSliceBytes,
                     kSliceBytes, &bar->w2_full[s]);
      }
    }
    __syncwarp();
  } else if (warp == 4) {
    // ---- MMA issue ----
    if ((tid & 31) == 0) {
      constexpr uint32_t kI256 = idesc_tf32(128, 256);
      constexpr uint32_t kI16 = idesc_tf32(128, 16);
      bool ok = true;
      for (int t = 0; t < steps && ok; ++t) {
        const uint32_t ph = (uint32_t)t & 1u;
        if (!(ok = tc::mbar_wait(&bar->obs_full, ph, abort, kWaitLimitNs))) break;
        tc::tc_fence_after();
        // K = 24 covers the 18 observation columns (the rest of the tile and
        // of W1 is zero)
        static_assert(kObs <= 24, "observation width");
#pragma unroll
        for (int kk = 0; kk < 3; ++kk)
          mma_ss(tmem, desc(s_base + kSObs + kk * 32), desc(s_base + kSW1 + kk * 32), kI256,
                 kk > 0 ? 1u : 0u);
        tc::mma_commit(&bar->l1_full);
        // layer 2, K-slice by K-slice as the epilogue writes h1's chunks
        for (int j = 0; j < kSlices && ok; ++j) {
          const int g = t * kSlices + j, s = g % kRing;
          if (!(ok = tc::mbar_wait(&bar->h1_part[j], ph, abort, kWaitLimitNs))) break;
          if (!(ok = tc::mbar_wait(&bar->w2_full[s], (uint32_t)(g / kRing) & 1u, abort,
                                   kWaitLimitNs)))
            break;
          tc::tc_fence_after();
          const uint32_t b0 = s_base + kSRing + s * kSliceBytes;
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            mma_ts(tmem + 256, tmem + 32 * j + 8 * kk, desc(b0 + kk * 32), kI256,
                   (j > 0 || kk > 0) ? 1u : 0u);
          tc::mma_commit(&bar->w2_empty[s]);
        }
        if (!ok) break;
        tc::mma_commit(&bar->l2_full);
        for (int j = 0; j < kSlices && ok; ++j) {
          if (!(ok = tc::mbar_wait(&bar->h2_part[j], ph, abort, kWaitLimitNs))) break;
          tc::tc_fence_after();
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            mma_ts(tmem, tmem + 256 + 32 * j + 8 * kk, desc(s_base + kSW3 + j * kW3Slice + kk * 32),
                   kI16, (j > 0 || kk > 0) ? 1u : 0u);
        }
        if (!ok) break;
        tc::mma_commit(&bar->l3_full);
      }
      tc::mma_commit(&bar->drain);
      tc::mbar_wait(&bar->drain, 0, abort, kWaitLimitNs);
    }
    __syncwarp();
  } else {
    // ---- env threads: observation, epilogues, sampling, physics ----
    const int row = tid;
    const int i = blockIdx.x * kRows + row;
    const bool active = i < M.n;
    const size_t n = (size_t)M.n;
    const uint32_t lane_addr = tmem + ((uint32_t)(warp * 32) << 16);
    const float* bias = reinterpret_cast<const float*>(smem + kSB);
    uint8_t* obs_tile = smem + kSObs;
    Env e;
    if (active) load_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
    bool bad = false, ok = true;
    for (int t = 0; t < steps && ok; ++t) {
      const uint32_t ph = (uint32_t)t & 1u;
      float o[kObs];
      if (active) {
        observe(e, o);
        if (tr.obs) {
#pragma unroll
          for (int k = 0; k < kObs; ++k) tr.obs[((size_t)t * kObs + k) * n + i] = o[k];
        }
      } else {
#pragma unroll
        for (int k = 0; k < kObs; ++k) o[k] = 0.0f;
      }
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        float4 v;
        v.x = 4 * q + 0 < kObs ? to_tf32(o[4 * q + 0]) : 0.0f;
        v.y = 4 * q + 1 < kObs ? to_tf32(o[4 * q + 1]) : 0.0f;
        v.z = 4 * q + 2 < kObs ? to_tf32(o[4 * q + 2]) : 0.0f;
        v.w = 4 * q + 3 < kObs ? to_tf32(o[4 * q + 3]) : 0.0f;
        *reinterpret_cast<float4*>(obs_tile + row * 128 + ((q ^ (row & 7)) << 4)) = v;
      }
      tc::fence_async_smem();
      tc::mbar_arrive(&bar->obs_full);
      __syncwarp();
      if (!(ok = tc::mbar_wait(&bar->l1_full, ph, abort, kWaitLimitNs))) break;
      tc::tc_fence_after();
      hidden_epilogue(lane_addr, 0, bias, bar->h1_part);
      // The step's normals depend only on (env, seed, step): drawn here,
      // while layer 2's last MMAs run, instead of after the head.
      const uint32_t id = M.id_base + (uint32_t)i;
      float eps[kAct];
      if (active) action_noise(id, M.seed, t_g0 + (uint64_t)t, eps);
      if (!(ok = tc::mbar_wait(&bar->l2_full, ph, abort, kWaitLimitNs))) break;
      tc::tc_fence_after();
      hidden_epilogue(lane_addr, 256, bias + kH, bar->h2_part);
      if (!(ok = tc::mbar_wait(&bar->l3_full, ph, abort, kWaitLimitNs))) break;
      tc::tc_fence_after();
      uint32_t o3[16];
      tc::tmem_ld16(lane_addr, o3);
      tc::tmem_ld_wait(o3);
      tc::tc_fence_before();
      __syncwarp();
      if (active) {
        float head[16];
#pragma unroll
        for (int k = 0; k < 16; ++k) head[k] = __uint_as_float(o3[k]) + bias[2 * kH + k];
        float a[kAct], lp;
        sample(M, head, eps, a, &lp);
        if (tr.act) {
#pragma unroll
          for (int k = 0; k < kAct; ++k) tr.act[((size_t)t * kAct + k) * n + i] = a[k];
        }
        if (tr.logp) tr.logp[(size_t)t * n + i] = lp;
        bool d;
        const float r = physics_step(M, id, e, a, &d);
        if (tr.rew) tr.rew[(size_t)t * n + i] = r;
        if (tr.done) tr.done[(size_t)t * n + i] = d ? 1 : 0;
        bad |= !env_finite(e);
      }
      __syncwarp();
    }
    if (active) {
      if (bad) flag_nan(st, i);
      store_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
    }
  }
  tc::tc_fence_before();
  __syncthreads();
  if (tid == 0 && bar->abort) {
    atomicAdd(&st->timeouts, 1);
    atomicCAS(&st->code, 0, -4);
  }
  if (warp == 4) {
    tc::tc_fence_after();
    tc::tmem_dealloc(tmem, 512);
  }
}

// ---------------------------------------------------------------------------
// Small batches (at most one tile per two SMs): a cluster of two CTAs per
// tile.  Both CTAs hold W1, W3 and the biases, and each holds its half of W2
// (rows 128r..128r+127 of every K-slice: 128 KB, resident, no streaming).
// Both compute the observation, layer 1 and h1 for the same 128 envs; CTA r
// then computes columns 128r..128r+127 of layer 2, their epilogue and the
// partial head over them (K-slices 4r..4r+3 of W3), and the two partial
// heads are exchanged through distributed shared memory and summed in rank
// order, so both CTAs hold the same head and run the same sampling and
// physics (identical state); CTA 0 writes the trajectory.  A control step is
// one tile's serial chain either way; this halves its layer 2 and its
// layer-2 epilogue.
// ---------------------------------------------------------------------------
constexpr uint32_t kPHalf = kSliceBytes / 2;              // one K-slice, 128 rows
constexpr uint32_t kPSObs = kSObs;
constexpr uint32_t kPSW2 = kPSObs + kRows * 128;          // 8 half K-slices of W2
constexpr uint32_t kPSX = kPSW2 + kSlices * kPHalf;       // exchange: [2][128][16] fp32
constexpr uint32_t kPSBar = kPSX + 2 * kRows * 16 * 4;

struct PairBars {
  uint64_t img_full, obs_full, l1_full, l2_full, l3_full, drain;
  uint64_t h1_part[kSlices];   // h1 chunk j written (128 arrivals)
  uint64_t h2_part[4];         // h2 chunk j of this CTA's half written (128 arrivals)
  uint64_t xch_full[2];        // the other CTA's partial head in exchange slot s (128 arrivals)
  uint32_t tmem_base;
  int abort;
};
constexpr uint32_t kPSmem = kPSBar + sizeof(PairBars) + 1024;
static_assert(kPSmem <= 227u * 1024u, "shared memory per CTA");
constexpr uint32_t kColHalf = 256;   // this CTA's 128 columns of layer 2, then h2
constexpr uint32_t kColPart = 384;   // partial head (16 columns)

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(160, 1)
k_rollout_tf32_pair(const Model M, Buffers B, const uint8_t* __restrict__ image, Traj tr, int T,
                    uint64_t t_g0, Status* st) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023u) & ~(uintptr_t)1023u);
  PairBars* bar = reinterpret_cast<PairBars*>(smem + kPSBar);
  volatile int* abort = &bar->abort;
  const int tid = threadIdx.x, warp = tid >> 5;
  const uint32_t rank = tc::cluster_rank(), peer = rank ^ 1u;

  if (tid == 0) {
    tc::mbar_init(&bar->img_full, 1);
    tc::mbar_init(&bar->obs_full, kRows);
    tc::mbar_init(&bar->l1_full, 1);
    tc::mbar_init(&bar->l2_full, 1);
    tc::mbar_init(&bar->l3_full, 1);
    tc::mbar_init(&bar->drain, 1);
    for (int j = 0; j < kSlices; ++j) tc::mbar_init(&bar->h1_part[j], kRows);
    for (int j = 0; j < 4; ++j) tc::mbar_init(&bar->h2_part[j], kRows);
    tc::mbar_init(&bar->xch_full[0], kRows);
    tc::mbar_init(&bar->xch_full[1], kRows);
    bar->abort = 0;
    tc::mbar_fence_init();
    tc::mbar_arrive_expect_tx(&bar->img_full, kH * 128 + kSlices * kW3Slice + (2 * kH + 16) * 4 +
                                                  kSlices * kPHalf);
    tc::bulk_g2s(smem + kSW1, image + kOffW1, kH * 128, &bar->img_full);
    tc::bulk_g2s(smem + kSW3, image + kOffW3, kSlices * kW3Slice, &bar->img_full);
    tc::bulk_g2s(smem + kSB, image + kOffB, (2 * kH + 16) * 4, &bar->img_full);
    for (int j = 0; j < kSlices; ++j)
      tc::bulk_g2s(smem + kPSW2 + j * kPHalf, image + kOffW2 + j * kSliceBytes + rank * kPHalf,
                   kPHalf, &bar->img_full);
  }
  if (warp == 4) {
    tc::tmem_alloc(&bar->tmem_base, 512);
    tc::tmem_relinquish();
  }
  tc::tc_fence_before();
  // both CTAs' barriers exist before either arrives on the other's
  tc::cluster_sync();
  tc::tc_fence_after();
  const uint32_t tmem = bar->tmem_base;
  const uint32_t s_base = tc::smem_u32(smem);
  const bool img_ok = tc::mbar_wait(&bar->img_full, 0, abort, kWaitLimitNs);
  const int steps = img_ok ? T : 0;

  if (warp == 4) {
    // ---- MMA issue ----
    if ((tid & 31) == 0) {
      constexpr uint32_t kI256 = idesc_tf32(128, 256);
      constexpr uint32_t kI128 = idesc_tf32(128, 128);
      constexpr uint32_t kI16 = idesc_tf32(128, 16);
      bool ok = true;
      for (int t = 0; t < steps && ok; ++t) {
        const uint32_t ph = (uint32_t)t & 1u;
        if (!(ok = tc::mbar_wait(&bar->obs_full, ph, abort, kWaitLimitNs))) break;
        tc::tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < 3; ++kk)   // K = 24 covers the 18 observation columns
          mma_ss(tmem, desc(s_base + kPSObs + kk * 32), desc(s_base + kSW1 + kk * 32), kI256,
                 kk > 0 ? 1u : 0u);
        tc::mma_commit(&bar->l1_full);
        // this CTA's half of layer 2, K-slice by K-slice as h1's chunks land
        for (int j = 0; j < kSlices && ok; ++j) {
          if (!(ok = tc::mbar_wait(&bar->h1_part[j], ph, abort, kWaitLimitNs))) break;
          tc::tc_fence_after();
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            mma_ts(tmem + kColHalf, tmem + 32 * j + 8 * kk,
                   desc(s_base + kPSW2 + j * kPHalf + kk * 32), kI128, (j > 0 || kk > 0) ? 1u : 0u);
        }
        if (!ok) break;
        tc::mma_commit(&bar->l2_full);
        // the partial head over this half's h2 chunks (W3 K-slices 4r + j)
        for (int j = 0; j < 4 && ok; ++j) {
          if (!(ok = tc::mbar_wait(&bar->h2_part[j], ph, abort, kWaitLimitNs))) break;
          tc::tc_fence_after();
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            mma_ts(tmem + kColPart, tmem + kColHalf + 32 * j + 8 * kk,
                   desc(s_base + kSW3 + (4 * rank + j) * kW3Slice + kk * 32), kI16,
                   (j > 0 || kk > 0) ? 1u : 0u);
        }
        if (!ok) break;
        tc::mma_commit(&bar->l3_full);
      }
      tc::mma_commit(&bar->drain);
      tc::mbar_wait(&bar->drain, 0, abort, kWaitLimitNs);
    }
    __syncwarp();
  } else {
    // ---- env threads (both CTAs; CTA 0 writes the trajectory) ----
    const int row = tid;
    const int i = (int)(blockIdx.x >> 1) * kRows + row;
    const bool active = i < M.n, writer = rank == 0;
    const size_t n = (size_t)M.n;
    const uint32_t lane_addr = tmem + ((uint32_t)(warp * 32) << 16);
    const float* bias = reinterpret_cast<const float*>(smem + kSB);
    uint8_t* obs_tile = smem + kPSObs;
    float* xch = reinterpret_cast<float*>(smem + kPSX);
    Env e;
    if (active) load_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
    bool bad = false, ok = true;
    for (int t = 0; t < steps && ok; ++t) {
      const uint32_t ph = (uint32_t)t & 1u;
      float o[kObs];
      if (active) {
        observe(e, o);
        if (writer && tr.obs) {
#pragma unroll
          for (int k = 0; k < kObs; ++k) tr.obs[((size_t)t * kObs + k) * n + i] = o[k];
        }
      } else {
#pragma unroll
        for (int k = 0; k < kObs; ++k) o[k] = 0.0f;
      }
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        float4 v;
        v.x = 4 * q + 0 < kObs ? to_tf32(o[4 * q + 0]) : 0.0f;
        v.y = 4 * q + 1 < kObs ? to_tf32(o[4 * q + 1]) : 0.0f;
        v.z = 4 * q + 2 < kObs ? to_tf32(o[4 * q + 2]) : 0.0f;
        v.w = 4 * q + 3 < kObs ? to_tf32(o[4 * q + 3]) : 0.0f;
        *reinterpret_cast<float4*>(obs_tile + row * 128 + ((q ^ (row & 7)) << 4)) = v;
      }
      tc::fence_async_smem();
      tc::mbar_arrive(&bar->obs_full);
      __syncwarp();
      if (!(ok = tc::mbar_wait(&bar->l1_full, ph, abort, kWaitLimitNs))) break;
      tc::tc_fence_after();
      hidden_epilogue(lane_addr, 0, bias, bar->h1_part);
      const uint32_t id = M.id_base + (uint32_t)i;
      float eps[kAct];
      if (active) action_noise(id, M.seed, t_g0 + (uint64_t)t, eps);
      if (!(ok = tc::mbar_wait(&bar->l2_full, ph, abort, kWaitLimitNs))) break;
      tc::tc_fence_after();
      // this CTA's 128 columns of h2: four chunks, each announced to layer 3
#pragma unroll 1
      for (int c = 0; c < 4; ++c) {
        uint32_t acc[32];
        const float* b2 = bias + kH + 128 * rank + 32 * c;
        tc::tmem_ld32(lane_addr + kColHalf + 32 * c, acc);
        tc::tmem_ld_wait(acc);
#pragma unroll
        for (int j = 0; j < 32; ++j)
          acc[j] = __float_as_uint(to_tf32(tc::tanh_f32(__uint_as_float(acc[j]) + b2[j])));
        tmem_st32(lane_addr + kColHalf + 32 * c, acc);
        tc::tmem_st_wait();
        tc::tc_fence_before();
        tc::mbar_arrive(&bar->h2_part[c]);
      }
      if (!(ok = tc::mbar_wait(&bar->l3_full, ph, abort, kWaitLimitNs))) break;
      tc::tc_fence_after();
      uint32_t p3[16];
      tc::tmem_ld16(lane_addr + kColPart, p3);
      tc::tmem_ld_wait(p3);
      tc::tc_fence_before();
      // the partial head to the other CTA's exchange slot t & 1, then its
      // arrival there; then the other CTA's partial from this CTA's slot
      const uint32_t slot = (uint32_t)t & 1u;
      const uint32_t xoff = tc::smem_u32(xch + (slot * kRows + row) * 16);
      const uint32_t xrem = tc::mapa(xoff, peer);
#pragma unroll
      for (int q = 0; q < 4; ++q)
        tc::st_cluster_v4(xrem + 16 * q, __uint_as_float(p3[4 * q]), __uint_as_float(p3[4 * q + 1]),
                          __uint_as_float(p3[4 * q + 2]), __uint_as_float(p3[4 * q + 3]));
      tc::mbar_arrive_cluster(tc::mapa(tc::smem_u32(&bar->xch_full[slot]), peer));
      if (!(ok = tc::mbar_wait_cluster(&bar->xch_full[slot], ((uint32_t)t >> 1) & 1u, abort,
                                       kWaitLimitNs)))
        break;
      __syncwarp();
      if (active) {
        const float* other = xch + (slot * kRows + row) * 16;
        float head[16];
        // CTA 0's partial plus CTA 1's (the same sum in both CTAs), + b3
#pragma unroll
        for (int k = 0; k < 16; ++k)
          head[k] = (__uint_as_float(p3[k]) + other[k]) + bias[2 * kH + k];
        float a[kAct], lp;
        sample(M, head, eps, a, &lp);
        if (writer) {
          if (tr.act) {
#pragma unroll
            for (int k = 0; k < kAct; ++k) tr.act[((size_t)t * kAct + k) * n + i] = a[k];
          }
          if (tr.logp) tr.logp[(size_t)t * n + i] = lp;
        }
        bool d;
        const float r = physics_step(M, id, e, a, &d);
        if (writer) {
          if (tr.rew) tr.rew[(size_t)t * n + i] = r;
          if (tr.done) tr.done[(size_t)t * n + i] = d ? 1 : 0;
        }
        bad |= !env_finite(e);
      }
      __syncwarp();
    }
    if (active && writer) {
      if (bad) flag_nan(st, i);
      store_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
    }
  }
  tc::tc_fence_before();
  __syncthreads();
  if (tid == 0 && bar->abort) {
    atomicAdd(&st->timeouts, 1);
    atomicCAS(&st->code, 0, -4);
  }
  // neither CTA leaves while the other may still write into its shared memory
  tc::cluster_sync();
  if (warp == 4) {
    tc::tc_fence_after();
    tc::tmem_dealloc(tmem, 512);
  }
}

}  // namespace

size_t tf32_policy_image_bytes() { return kImage; }

cudaError_t launch_pack_tf32(const Model& M, const float* wp_f32, void* packed, cudaStream_t s) {
  const int pieces = kH * 32 + kH * kH + kSlices * 16 * 32 + 2 * kH + 16;
  k_pack_tf32<<<(pieces + 255) / 256, 256, 0, s>>>(wp_f32, kObs, M.policy_out,
                                                   static_cast<uint8_t*>(packed));
  return cudaGetLastError();
}

cudaError_t launch_rollout_tf32(const Model& M, const Buffers& B, const void* packed,
                                const Traj& tr, int T, uint64_t t_g0, Status* st, cudaStream_t s) {
  cudaError_t e = cudaFuncSetAttribute(k_rollout_tf32, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)kSmem);
  if (e != cudaSuccess) return e;
  const int grid = (M.n + kRows - 1) / kRows;
  if (2 * grid <= engine_sm_count()) {
    // at most one tile per two SMs: the two-CTA kernel
    e = cudaFuncSetAttribute(k_rollout_tf32_pair, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)kPSmem);
    if (e != cudaSuccess) return e;
    k_rollout_tf32_pair<<<2 * grid, 160, kPSmem, s>>>(M, B, static_cast<const uint8_t*>(packed),
                                                      tr, T, t_g0, st);
    return cudaGetLastError();
  }
  k_rollout_tf32<<<grid, 192, kSmem, s>>>(M, B, static_cast<const uint8_t*>(packed), tr, T, t_g0,
                                          st);
  return cudaGetLastError();
}

}  // namespace auv
