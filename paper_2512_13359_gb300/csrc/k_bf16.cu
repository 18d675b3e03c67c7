// k_bf16.cu -- tensor-core network engine of the batched AUV rollout.
//
// Networks (hidden width 256, tanh): the policy 18 -> 256 -> 256 -> 16 (mean,
// log-std) and the value 18 -> 256 -> 256 -> 1, bf16 weights and activations,
// fp32 accumulation in tensor memory (tcgen05.mma kind::f16), fp32 biases.
//
// One CTA per SM holds the network's weights in shared memory as pre-swizzled
// bf16 images for the whole launch.  Its threads form G groups of 128 (one
// row -- one environment -- per thread, which is also that row's tensor-memory
// lane) plus one MMA-issuing warp.  The groups take turns on the tensor pipe:
// while one group's network runs, the others integrate their environments.
//
// Per 128-row tile and control step:
//   layer 1: A = observation tile (smem, K = 32 with 18 used), 4 N-chunks of 64
//   epilogue: + b1, tanh, bf16 -> h1 written back to tensor memory
//   layer 2: A = h1 from tensor memory (K = 256), 4 N-chunks of 64
//   epilogue: + b2, tanh, bf16 -> h2 chunk in smem (policy), or the value
//             head's dot product on CUDA cores (value)
//   layer 3 (policy): A = h2 chunk (smem), B = W3 K-slice, accumulated over
//             the 4 chunks into a 16-column fp32 accumulator
//
// Tensor-memory columns: acc[0] 0..63, acc[1] 64..127, h1 128..255 (bf16
// pairs), acc3 256..271.
#include <climits>

#include "auv_bf16.h"
#include "tc_ptx.cuh"

namespace auv {

namespace {

constexpr int kH = 256;
constexpr int kRows = 128;
constexpr int kChunk = 64;
constexpr int kNChunks = kH / kChunk;
constexpr int kHeadOut = 16;

// Packed image (bytes).  W1: 256 rows x 64 B (K = 32), 64-byte swizzle.
// W2: 4 K-atoms x 256 rows x 128 B, 128-byte swizzle.  W3: 4 K-atoms x 16
// rows x 128 B.  Then fp32 b1[256], b2[256] and either b3[16] (policy) or
// w3[256] (bf16-rounded) and b3[1] (value).
constexpr uint32_t kW1Bytes = kH * 64;
constexpr uint32_t kW2Bytes = 4 * kH * 128;
constexpr uint32_t kW3Bytes = 4 * kHeadOut * 128;
constexpr uint32_t kOffW1 = 0;
constexpr uint32_t kOffW2 = kOffW1 + kW1Bytes;
constexpr uint32_t kOffW3 = kOffW2 + kW2Bytes;
constexpr uint32_t kOffB1P = kOffW3 + kW3Bytes;
constexpr uint32_t kOffB2P = kOffB1P + kH * 4;
constexpr uint32_t kOffB3P = kOffB2P + kH * 4;
constexpr uint32_t kPolicyImage = kOffB3P + 256;
constexpr uint32_t kOffB1V = kOffW2 + kW2Bytes;
constexpr uint32_t kOffB2V = kOffB1V + kH * 4;
constexpr uint32_t kOffW3V = kOffB2V + kH * 4;
constexpr uint32_t kOffB3V = kOffW3V + kH * 4;
constexpr uint32_t kValueImage = kOffB3V + 256;

constexpr uint32_t kObsTileBytes = kRows * 64;    // SW64, K = 32
constexpr uint32_t kH2TileBytes = kRows * 128;    // SW128, K = 64

constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColAcc0 = 0, kColAcc1 = 64, kColH1 = 128, kColAcc3 = 256;

constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s per wait

enum Mode { kRollout = 0, kPolicyRows = 1, kValueRows = 2 };

// -------------------------------------------------------------------------
// weight packing
// -------------------------------------------------------------------------
__device__ __forceinline__ uint16_t bf16_bits(float x) {
  return (uint16_t)(tc::pack_bf16x2(x, 0.0f) & 0xFFFFu);
}

// One thread per 16-byte piece of the W1/W2/W3 regions, then the vectors.
__global__ void k_pack(const float* __restrict__ w, int out_dim, uint8_t* __restrict__ img) {
  const int kObsDim = 18;
  const float* W1 = w;
  const float* b1 = W1 + kH * kObsDim;
  const float* W2 = b1 + kH;
  const float* b2 = W2 + kH * kH;
  const float* W3 = b2 + kH;
  const float* b3 = W3 + out_dim * kH;
  const bool policy = out_dim == kHeadOut;
  const int n_w1 = kH * 4, n_w2 = 4 * kH * 8, n_w3 = policy ? 4 * kHeadOut * 8 : 0;
  const int piece = blockIdx.x * blockDim.x + threadIdx.x;
  uint16_t v[8];
  uint32_t off;
  if (piece < n_w1) {
    const int n = piece >> 2, p = piece & 3, q = p ^ ((n >> 1) & 3);
    for (int e = 0; e < 8; ++e) {
      const int k = 8 * q + e;
      v[e] = k < kObsDim ? bf16_bits(W1[n * kObsDim + k]) : (uint16_t)0;
    }
    off = kOffW1 + n * 64 + p * 16;
  } else if (piece < n_w1 + n_w2) {
    const int id = piece - n_w1;
    const int a = id / (kH * 8), n = (id / 8) % kH, p = id & 7, q = p ^ (n & 7);
    for (int e = 0; e < 8; ++e) v[e] = bf16_bits(W2[n * kH + 64 * a + 8 * q + e]);
    off = kOffW2 + a * (kH * 128) + n * 128 + p * 16;
  } else if (piece < n_w1 + n_w2 + n_w3) {
    const int id = piece - n_w1 - n_w2;
    const int a = id / (kHeadOut * 8), n = (id / 8) % kHeadOut, p = id & 7, q = p ^ (n & 7);
    for (int e = 0; e < 8; ++e) v[e] = bf16_bits(W3[n * kH + 64 * a + 8 * q + e]);
    off = kOffW3 + a * (kHeadOut * 128) + n * 128 + p * 16;
  } else {
    const int id = piece - n_w1 - n_w2 - n_w3;   // vector entries, one float each
    float* f = reinterpret_cast<float*>(img);
    if (policy) {
      if (id < kH) f[(kOffB1P >> 2) + id] = b1[id];
      else if (id < 2 * kH) f[(kOffB2P >> 2) + id - kH] = b2[id - kH];
      else if (id < 2 * kH + kHeadOut) f[(kOffB3P >> 2) + id - 2 * kH] = b3[id - 2 * kH];
    } else {
      if (id < kH) f[(kOffB1V >> 2) + id] = b1[id];
      else if (id < 2 * kH) f[(kOffB2V >> 2) + id - kH] = b2[id - kH];
      else if (id < 3 * kH)
        f[(kOffW3V >> 2) + id - 2 * kH] = __uint_as_float((uint32_t)bf16_bits(W3[id - 2 * kH]) << 16);
      else if (id == 3 * kH) f[kOffB3V >> 2] = b3[0];
    }
    return;
  }
  uint4 pk;
  pk.x = v[0] | ((uint32_t)v[1] << 16);
  pk.y = v[2] | ((uint32_t)v[3] << 16);
  pk.z = v[4] | ((uint32_t)v[5] << 16);
  pk.w = v[6] | ((uint32_t)v[7] << 16);
  *reinterpret_cast<uint4*>(img + off) = pk;
}

// -------------------------------------------------------------------------
// engine
// -------------------------------------------------------------------------
struct Barriers {
  uint64_t obs_full[4];
  uint64_t acc_full[4][2];
  uint64_t acc3_full[4];
  uint64_t acc_empty[2];
  uint64_t h2_full[2];
  uint64_t acc3_empty;
  uint64_t h1_full;
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
};

struct RowIO {            // row modes: obs element (r, k) at ((r / ns) * 18 + k) * ns + r % ns
  const float* obs;
  size_t rows;
  int ns;
  float* out;             // head[r][16] (policy) or value[r] (value)
};

template <int G, int MODE>
struct Engine {
  static constexpr bool kPolicy = MODE != kValueRows;
  static constexpr uint32_t kImage = kPolicy ? kPolicyImage : kValueImage;
  static constexpr uint32_t kImageAl = (kImage + 1023u) & ~1023u;
  static constexpr uint32_t kOffObs = kImageAl;
  static constexpr uint32_t kOffH2 = kOffObs + G * kObsTileBytes;
  static constexpr uint32_t kOffBar = kOffH2 + (kPolicy ? 2 * kH2TileBytes : 0);
  static constexpr uint32_t kSmem = kOffBar + sizeof(Barriers) + 1024;   // + alignment slack
  static constexpr int kThreads = G * kRows + 32;
};

// Row r of the observation tile (bf16, K = 32, 64-byte swizzle): 4 pieces of
// 16 bytes, piece q at position q ^ ((r >> 1) & 3).  Features 18..31 are zero.
__device__ __forceinline__ void write_obs_row(uint8_t* tile, int r, const float o[kObs]) {
  uint32_t w[16];
#pragma unroll
  for (int j = 0; j < 9; ++j) w[j] = tc::pack_bf16x2(o[2 * j], o[2 * j + 1]);
#pragma unroll
  for (int j = 9; j < 16; ++j) w[j] = 0u;
  const int sw = (r >> 1) & 3;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    uint4 v = make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
    *reinterpret_cast<uint4*>(tile + r * 64 + ((q ^ sw) << 4)) = v;
  }
}

// 32 accumulator columns + bias -> tanh -> 16 bf16 pairs.
__device__ __forceinline__ void bias_tanh32(const uint32_t (&acc)[32], const float* bias,
                                            uint32_t (&out)[16]) {
#pragma unroll
  for (int j = 0; j < 16; j += 2) {
    const float4 b = *reinterpret_cast<const float4*>(bias + 2 * j);
    out[j] = tc::tanh_bf16x2(tc::pack_bf16x2(__uint_as_float(acc[2 * j]) + b.x,
                                             __uint_as_float(acc[2 * j + 1]) + b.y));
    out[j + 1] = tc::tanh_bf16x2(tc::pack_bf16x2(__uint_as_float(acc[2 * j + 2]) + b.z,
                                                 __uint_as_float(acc[2 * j + 3]) + b.w));
  }
}

// Register cap: the 4G+1 warps are spread over the SM's four sub-partitions,
// whose 16K-register files each host G+1 warps (G = 4: 5 warps x 32 lanes
// x 96 registers <= 16384).
template <int G, int MODE>
__global__ void __launch_bounds__(G * 128 + 32) __maxnreg__(G == 4 ? 96 : 168)
k_engine(const Model M, Buffers B, const uint8_t* __restrict__ image, Traj tr, int T,
         uint64_t t_g0, RowIO io, Status* st) {
  using E = Engine<G, MODE>;
  constexpr bool kPolicy = E::kPolicy;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023u) & ~(uintptr_t)1023u);
  Barriers* bar = reinterpret_cast<Barriers*>(smem + E::kOffBar);
  volatile int* abort = &bar->abort;
  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const bool is_mma_warp = warp == 4 * G;

  // ---- set-up: barriers, weights, tensor memory ----
  if (tid == 0) {
    for (int g = 0; g < G; ++g) {
      tc::mbar_init(&bar->obs_full[g], kRows);
      tc::mbar_init(&bar->acc_full[g][0], 1);
      tc::mbar_init(&bar->acc_full[g][1], 1);
      tc::mbar_init(&bar->acc3_full[g], 1);
    }
    tc::mbar_init(&bar->acc_empty[0], kRows);
    tc::mbar_init(&bar->acc_empty[1], kRows);
    tc::mbar_init(&bar->h2_full[0], kRows);
    tc::mbar_init(&bar->h2_full[1], kRows);
    tc::mbar_init(&bar->acc3_empty, kRows);
    tc::mbar_init(&bar->h1_full, kRows);
    tc::mbar_init(&bar->drain, 1);
    bar->abort = 0;
    tc::mbar_fence_init();
  }
  {
    const uint4* src = reinterpret_cast<const uint4*>(image);
    uint4* dst = reinterpret_cast<uint4*>(smem);
    for (uint32_t i = tid; i < E::kImage / 16; i += blockDim.x) dst[i] = __ldg(src + i);
  }
  tc::fence_async_smem();
  if (is_mma_warp) {
    tc::tmem_alloc(&bar->tmem_base, kTmemCols);
    tc::tmem_relinquish();
  }
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = bar->tmem_base;
  const uint32_t s_base = tc::smem_u32(smem);

  // ---- work assignment ----
  const int n_tiles = MODE == kRollout ? (M.n + kRows - 1) / kRows
                                       : (int)((io.rows + kRows - 1) / kRows);
  const int slot0 = blockIdx.x * G;
  const int n_slots = gridDim.x * G;
  auto group_iters = [&](int g) -> int {
    const int s = slot0 + g;
    if (MODE == kRollout) return s < n_tiles ? T : 0;
    return s < n_tiles ? (n_tiles - s - 1) / n_slots + 1 : 0;
  };

  if (is_mma_warp) {
    // =================== MMA issue (one elected lane) ===================
    if ((tid & 31) == 0) {
      constexpr uint32_t kI64 = tc::idesc_bf16_f32(128, kChunk);
      constexpr uint32_t kI16 = tc::idesc_bf16_f32(128, kHeadOut);
      const uint32_t tacc[2] = {tmem + kColAcc0, tmem + kColAcc1};
      uint32_t use_acc[2] = {0, 0}, use_h1 = 0, use_h2[2] = {0, 0}, use_acc3 = 0;
      uint32_t obs_phase[4] = {0, 0, 0, 0};
      int max_iters = 0;
      for (int g = 0; g < G; ++g) max_iters = max(max_iters, group_iters(g));
      bool ok = true;
      auto acquire_acc = [&](int b) -> bool {
        const bool r = tc::mbar_wait(&bar->acc_empty[b], (use_acc[b] & 1u) ^ 1u, abort,
                                     kWaitLimitNs);
        ++use_acc[b];
        tc::tc_fence_after();
        return r;
      };
      auto issue_l2 = [&](int g, int c) -> bool {
        const int b = c & 1;
        if (!acquire_acc(b)) return false;
#pragma unroll 1
        for (int kk = 0; kk < 16; ++kk) {
          const uint64_t bd = tc::smem_desc(
              s_base + kOffW2 + (kk >> 2) * (kH * 128) + c * kChunk * 128 + (kk & 3) * 32, 1024, 2);
          tc::mma_ts(tacc[b], tmem + kColH1 + kk * 8, bd, kI64, kk > 0 ? 1u : 0u);
        }
        tc::mma_commit(&bar->acc_full[g][b]);
        return true;
      };
      for (int it = 0; it < max_iters && ok; ++it) {
        for (int g = 0; g < G && ok; ++g) {
          if (it >= group_iters(g)) continue;
          // layer 1
          ok = tc::mbar_wait(&bar->obs_full[g], obs_phase[g] & 1u, abort, kWaitLimitNs);
          ++obs_phase[g];
          if (!ok) break;
          tc::tc_fence_after();
          const uint32_t obs_s = s_base + E::kOffObs + g * kObsTileBytes;
          for (int c = 0; c < kNChunks && ok; ++c) {
            const int b = c & 1;
            if (!(ok = acquire_acc(b))) break;
#pragma unroll
            for (int kk = 0; kk < 2; ++kk) {
              const uint64_t ad = tc::smem_desc(obs_s + kk * 32, 512, 4);
              const uint64_t bd = tc::smem_desc(s_base + kOffW1 + c * kChunk * 64 + kk * 32, 512, 4);
              tc::mma_ss(tacc[b], ad, bd, kI64, kk);
            }
            tc::mma_commit(&bar->acc_full[g][b]);
          }
          if (!ok) break;
          // layer 2 needs the whole of h1
          ok = tc::mbar_wait(&bar->h1_full, use_h1 & 1u, abort, kWaitLimitNs);
          ++use_h1;
          if (!ok) break;
          tc::tc_fence_after();
          if (!kPolicy) {
            for (int c = 0; c < kNChunks && ok; ++c) ok = issue_l2(g, c);
            continue;
          }
          ok = issue_l2(g, 0) && issue_l2(g, 1);
          if (!ok) break;
          // layer 3 interleaved with the last two layer-2 chunks
          ok = tc::mbar_wait(&bar->acc3_empty, (use_acc3 & 1u) ^ 1u, abort, kWaitLimitNs);
          ++use_acc3;
          for (int c = 0; c < kNChunks && ok; ++c) {
            const int hb = c & 1;
            ok = tc::mbar_wait(&bar->h2_full[hb], use_h2[hb] & 1u, abort, kWaitLimitNs);
            ++use_h2[hb];
            if (!ok) break;
            tc::tc_fence_after();
            const uint32_t h2_s = s_base + E::kOffH2 + hb * kH2TileBytes;
#pragma unroll
            for (int kk = 0; kk < 4; ++kk) {
              const uint64_t ad = tc::smem_desc(h2_s + kk * 32, 1024, 2);
              const uint64_t bd = tc::smem_desc(s_base + kOffW3 + c * (kHeadOut * 128) + kk * 32,
                                                1024, 2);
              tc::mma_ss(tmem + kColAcc3, ad, bd, kI16, (c > 0 || kk > 0) ? 1u : 0u);
            }
            if (c == kNChunks - 1) tc::mma_commit(&bar->acc3_full[g]);
            if (c + 2 < kNChunks) ok = issue_l2(g, c + 2);
          }
        }
      }
      // drain: every issued MMA has completed before tensor memory is freed
      tc::mma_commit(&bar->drain);
      tc::mbar_wait(&bar->drain, 0, abort, kWaitLimitNs);
    }
    __syncwarp();
  } else {
    // =================== groups: epilogues + physics / row I/O ===================
    const int g = warp >> 2;
    const int row = tid & (kRows - 1);
    const uint32_t lane_addr = tmem + ((uint32_t)((warp & 3) * 32) << 16);
    uint8_t* obs_tile = smem + E::kOffObs + g * kObsTileBytes;
    uint8_t* h2_tiles = smem + E::kOffH2;
    const float* b1 = reinterpret_cast<const float*>(smem + (kPolicy ? kOffB1P : kOffB1V));
    const float* b2 = reinterpret_cast<const float*>(smem + (kPolicy ? kOffB2P : kOffB2V));
    uint32_t n_full[2] = {0, 0}, n_acc3 = 0;
    bool ok = true;

    auto wait_acc = [&](int b) -> bool {
      const bool r = tc::mbar_wait(&bar->acc_full[g][b], n_full[b] & 1u, abort, kWaitLimitNs);
      ++n_full[b];
      tc::tc_fence_after();
      return r;
    };
    // Layers 1 and 2 epilogues for this group's tile; value mode returns the
    // head dot product, policy mode leaves the 16 head outputs in head[].
    auto run_network = [&](float* head) -> bool {
      for (int c = 0; c < kNChunks; ++c) {       // layer 1 -> h1 (tensor memory)
        const int b = c & 1;
        if (!wait_acc(b)) return false;
        const uint32_t col = b ? kColAcc1 : kColAcc0;
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          uint32_t acc[32], hv[16];
          tc::tmem_ld32(lane_addr + col + 32 * half, acc);
          tc::tmem_ld_wait(acc);
          if (half == 1) {
            tc::tc_fence_before();
            tc::mbar_arrive(&bar->acc_empty[b]);
          }
          bias_tanh32(acc, b1 + c * kChunk + 32 * half, hv);
          tc::tmem_st16(lane_addr + kColH1 + c * 32 + half * 16, hv);
        }
      }
      tc::tmem_st_wait();
      tc::tc_fence_before();
      tc::mbar_arrive(&bar->h1_full);
      float vsum = 0.0f;
      const float* w3v = reinterpret_cast<const float*>(smem + kOffW3V);
      for (int c = 0; c < kNChunks; ++c) {       // layer 2
        const int b = c & 1;
        if (!wait_acc(b)) return false;
        const uint32_t col = b ? kColAcc1 : kColAcc0;
        uint8_t* h2 = h2_tiles + b * kH2TileBytes + row * 128;
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          uint32_t acc[32], hv[16];
          tc::tmem_ld32(lane_addr + col + 32 * half, acc);
          tc::tmem_ld_wait(acc);
          if (half == 1) {
            tc::tc_fence_before();
            tc::mbar_arrive(&bar->acc_empty[b]);
          }
          bias_tanh32(acc, b2 + c * kChunk + 32 * half, hv);
          if (kPolicy) {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const int pos = (4 * half + q) ^ (row & 7);
              *reinterpret_cast<uint4*>(h2 + (pos << 4)) =
                  make_uint4(hv[4 * q], hv[4 * q + 1], hv[4 * q + 2], hv[4 * q + 3]);
            }
          } else {
            const float* w = w3v + c * kChunk + 32 * half;
#pragma unroll
            for (int j = 0; j < 16; ++j)
              vsum = fmaf(tc::bf16lo(hv[j]), w[2 * j], fmaf(tc::bf16hi(hv[j]), w[2 * j + 1], vsum));
          }
        }
        if (kPolicy) {
          tc::fence_async_smem();
          tc::mbar_arrive(&bar->h2_full[b]);
        }
      }
      if (!kPolicy) {
        head[0] = vsum + *reinterpret_cast<const float*>(smem + kOffB3V);
        return true;
      }
      if (!tc::mbar_wait(&bar->acc3_full[g], n_acc3 & 1u, abort, kWaitLimitNs)) return false;
      ++n_acc3;
      tc::tc_fence_after();
      uint32_t o3[16];
      tc::tmem_ld16(lane_addr + kColAcc3, o3);
      tc::tmem_ld_wait(o3);
      tc::tc_fence_before();
      tc::mbar_arrive(&bar->acc3_empty);
      const float* b3 = reinterpret_cast<const float*>(smem + kOffB3P);
#pragma unroll
      for (int j = 0; j < kHeadOut; ++j) head[j] = __uint_as_float(o3[j]) + b3[j];
      return true;
    };

    const int iters = group_iters(g);
    if (MODE == kRollout) {
      const int tile = slot0 + g;
      const int i = tile * kRows + row;
      const bool active = iters > 0 && i < M.n;
      const size_t n = (size_t)M.n;
      Env e;
      if (active) load_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
      bool bad = false;
      for (int t = 0; t < iters && ok; ++t) {
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
        write_obs_row(obs_tile, row, o);
        tc::fence_async_smem();
        tc::mbar_arrive(&bar->obs_full[g]);
        float head[kHeadOut];
        __syncwarp();
        if (!(ok = run_network(head))) break;
        __syncwarp();
        if (active) {
          const uint32_t id = M.id_base + (uint32_t)i;
          float eps[kAct];
          action_noise(id, M.seed, t_g0 + (uint64_t)t, eps);
          float a[kAct], lp = 0.0f;
#pragma unroll
          for (int k = 0; k < kAct; ++k) {
            const float ls = fminf(fmaxf(head[kAct + k], M.logstd_min), M.logstd_max);
            a[k] = fmaf(expf(ls), eps[k], head[k]);
            lp += -0.5f * eps[k] * eps[k] - ls;
          }
          lp -= (float)kAct * 0.91893853320467274f;
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
    } else {
      for (int it = 0; it < iters && ok; ++it) {
        const size_t r = (size_t)(slot0 + g + it * n_slots) * kRows + row;
        const bool active = r < io.rows;
        float o[kObs];
        if (active) {
          const size_t ns = (size_t)io.ns;
          const size_t base = (r / ns) * kObs * ns + r % ns;
#pragma unroll
          for (int k = 0; k < kObs; ++k) o[k] = __ldg(io.obs + base + (size_t)k * ns);
        } else {
#pragma unroll
          for (int k = 0; k < kObs; ++k) o[k] = 0.0f;
        }
        write_obs_row(obs_tile, row, o);
        tc::fence_async_smem();
        tc::mbar_arrive(&bar->obs_full[g]);
        float head[kHeadOut];
        __syncwarp();
        if (!(ok = run_network(head))) break;
        __syncwarp();
        if (active) {
          if (MODE == kValueRows) {
            io.out[r] = head[0];
          } else {
#pragma unroll
            for (int k = 0; k < kHeadOut; ++k) io.out[r * kHeadOut + k] = head[k];
          }
        }
      }
    }
  }

  // ---- teardown ----
  __syncthreads();
  if (tid == 0 && bar->abort) {
    atomicAdd(&st->timeouts, 1);
    atomicCAS(&st->code, 0, -4);
  }
  if (is_mma_warp) {
    tc::tc_fence_after();
    tc::tmem_dealloc(tmem, kTmemCols);
  }
}

int sm_count() {
  static int cached = 0;
  if (!cached) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&cached, cudaDevAttrMultiProcessorCount, dev);
    if (cached <= 0) cached = 1;
  }
  return cached;
}

template <int G, int MODE>
cudaError_t launch_engine(int grid, const Model& M, const Buffers& B, const uint8_t* image,
                          const Traj& tr, int T, uint64_t t_g0, const RowIO& io, Status* st,
                          cudaStream_t s) {
  using E = Engine<G, MODE>;
  cudaError_t err = cudaFuncSetAttribute(k_engine<G, MODE>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, E::kSmem);
  if (err != cudaSuccess) return err;
  k_engine<G, MODE><<<grid, E::kThreads, E::kSmem, s>>>(M, B, image, tr, T, t_g0, io, st);
  return cudaGetLastError();
}

// Groups per CTA for `tiles` independent 128-row tiles on the SMs: fewest
// waves times groups (time per CTA grows with its groups); larger G on ties.
int pick_groups(long tiles) {
  const long sms = sm_count();
  int best = 4;
  long best_cost = LONG_MAX;
  for (int G = 4; G >= 1; G >>= 1) {
    const long ctas = (tiles + G - 1) / G;
    const long waves = (ctas + sms - 1) / sms;
    const long cost = waves * G;
    if (cost < best_cost) {
      best_cost = cost;
      best = G;
    }
  }
  return best;
}

}  // namespace

size_t bf16_policy_image_bytes() { return kPolicyImage; }
size_t bf16_value_image_bytes() { return kValueImage; }

cudaError_t launch_pack_bf16(const Model& M, const float* wp_f32, const float* wv_f32,
                             void* wp_packed, void* wv_packed, cudaStream_t s) {
  (void)M;
  const int pol_pieces = kH * 4 + 4 * kH * 8 + 4 * kHeadOut * 8 + 2 * kH + kHeadOut;
  k_pack<<<(pol_pieces + 255) / 256, 256, 0, s>>>(wp_f32, kHeadOut,
                                                  static_cast<uint8_t*>(wp_packed));
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess || !wv_f32) return e;
  const int val_pieces = kH * 4 + 4 * kH * 8 + 3 * kH + 1;
  k_pack<<<(val_pieces + 255) / 256, 256, 0, s>>>(wv_f32, 1, static_cast<uint8_t*>(wv_packed));
  return cudaGetLastError();
}

cudaError_t launch_rollout_bf16(const Model& M, const Buffers& B, const void* wp_packed,
                                const Traj& tr, int T, uint64_t t_g0, Status* st, cudaStream_t s) {
  const long tiles = (M.n + kRows - 1) / kRows;
  const int G = pick_groups(tiles);
  const int grid = (int)((tiles + G - 1) / G);
  const uint8_t* img = static_cast<const uint8_t*>(wp_packed);
  const RowIO io = {nullptr, 0, 1, nullptr};
  switch (G) {
    case 4: return launch_engine<4, kRollout>(grid, M, B, img, tr, T, t_g0, io, st, s);
    case 2: return launch_engine<2, kRollout>(grid, M, B, img, tr, T, t_g0, io, st, s);
    default: return launch_engine<1, kRollout>(grid, M, B, img, tr, T, t_g0, io, st, s);
  }
}

template <int MODE>
static cudaError_t launch_rows(const Model& M, const uint8_t* img, const RowIO& io, Status* st,
                               cudaStream_t s) {
  const long tiles = (long)((io.rows + kRows - 1) / kRows);
  const int G = tiles >= 4L * sm_count() ? 4 : (tiles >= 2L * sm_count() ? 2 : 1);
  const long want = (tiles + G - 1) / G;
  const int grid = (int)(want < sm_count() ? want : sm_count());
  const Buffers B = {nullptr, nullptr, nullptr, nullptr};
  const Traj tr = {nullptr, nullptr, nullptr, nullptr, nullptr, nullptr};
  switch (G) {
    case 4: return launch_engine<4, MODE>(grid, M, B, img, tr, 0, 0, io, st, s);
    case 2: return launch_engine<2, MODE>(grid, M, B, img, tr, 0, 0, io, st, s);
    default: return launch_engine<1, MODE>(grid, M, B, img, tr, 0, 0, io, st, s);
  }
}

cudaError_t launch_value_bf16(const Model& M, const void* wv_packed, const float* wv_f32,
                              const float* obs, size_t rows, int n, float* value, Status* st,
                              cudaStream_t s) {
  (void)wv_f32;
  const RowIO io = {obs, rows, n, value};
  return launch_rows<kValueRows>(M, static_cast<const uint8_t*>(wv_packed), io, st, s);
}

cudaError_t launch_forward_bf16(const Model& M, const void* wp_packed, const void* wv_packed,
                                const float* wv_f32, const float* obs, int n, float* head,
                                float* value, Status* st, cudaStream_t s) {
  (void)wv_f32;
  const RowIO io = {obs, (size_t)n, 1, head};
  cudaError_t e = launch_rows<kPolicyRows>(M, static_cast<const uint8_t*>(wp_packed), io, st, s);
  if (e != cudaSuccess || !value) return e;
  const RowIO iov = {obs, (size_t)n, 1, value};
  return launch_rows<kValueRows>(M, static_cast<const uint8_t*>(wv_packed), iov, st, s);
}

}  // namespace auv
