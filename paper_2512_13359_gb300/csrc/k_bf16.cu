// k_bf16.cu -- tensor-core network engine of the batched AUV rollout.
//
// Networks (hidden width 256, tanh): the policy 18 -> 256 -> 256 -> 16 (mean,
// log-std) and the value 18 -> 256 -> 256 -> 1, bf16 weights and activations,
// fp32 accumulation in tensor memory (tcgen05.mma kind::f16), fp32 biases.
//
// One CTA per SM holds the network's weights in shared memory as pre-swizzled
// bf16 images for the whole launch.  Its threads form G groups of 128 (one
// row -- one environment -- per thread, which is also that row's tensor-memory
// lane) plus three MMA-issuing warps (layer 1, layer 2, layer 3).  The groups take
// turns on the tensor pipe: while one group's network runs, the others
// integrate their environments.
//
// Per 128-row tile and control step:
//   layer 1: A = observation tile (smem, K = 32: the observation, zeros, and
//            ones in columns 30 and 31, which carry b1 as a bf16 hi + lo pair
//            in W1's columns 30 and 31), 4 N-chunks of 64
//   epilogue: tanh, bf16 -> h1 written back to tensor memory
//   layer 2: A = h1 from tensor memory (K = 256), 4 N-chunks of 64
//   epilogue: + b2, tanh, bf16 -> h2 chunk in smem (policy), or the value
//             head's dot product on CUDA cores (value)
//   layer 3 (policy): A = h2 chunk (smem), B = W3 K-slice, accumulated over
//             the 4 chunks into a 16-column fp32 accumulator
//
// Tensor-memory columns: h1 slots 0..127 and 128..255 (bf16 pairs), layer-1
// accumulator X 256..319, layer-2 accumulators Y 320..383 and Z 384..447,
// head accumulators 448..463 and 464..479.
//
// One group per CTA (the rollout with fewer tiles than SMs) differs: a
// second warpgroup takes the second 32-column half of every epilogue chunk;
// h1 stays in slot 0 while layer 1's chunks 0 and 1 accumulate in slot 1's
// columns, which then hold h2 (packed, layer 3's A operand from tensor
// memory); layer 2's chunks 0 and 1 start K-slice by K-slice as h1 is
// written.
#include <atomic>
#include <climits>

#include "auv_bf16.h"
#include "paper_device.cuh"
#include "tc_ptx.cuh"

namespace auv {

namespace {

constexpr int kH = 256;
constexpr int kRows = 128;
constexpr int kChunk = 64;
constexpr int kNChunks = kH / kChunk;
constexpr int kHeadOut = 16;

// Packed image (bytes).  W1: 256 rows x 64 B (K = 32: the input weights, zeros,
// then b1 split into bf16 hi and lo parts in columns 30 and 31), 64-byte swizzle.
// W2: 4 K-atoms x 256 rows x 128 B, 128-byte swizzle.  W3: 4 K-atoms x 16
// rows x 128 B.  Then fp32 b1[256] (layer 1 takes its bias through W1's
// columns 30 and 31 instead), b2[256] and either b3[16] (policy) or
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
constexpr uint32_t kColH1 = 0;      // two h1 slots of 128 columns (bf16 pairs)
constexpr uint32_t kColX = 256;     // layer-1 chunk accumulator (64 fp32 columns)
constexpr uint32_t kColY = 320;     // layer-2 even-chunk accumulator
constexpr uint32_t kColZ = 384;     // layer-2 odd-chunk accumulator
constexpr uint32_t kColA3 = 448;    // two head accumulators of 16 columns

constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s per wait

// Learner modes (compile-time, so that the plain row modes carry none of
// their code): kLearnPolicy / kLearnValue read bf16 input rows and also store
// H1 and H2; kBackRows is the backward-data pass, the engine's two layers on
// transposed weights (see k_pack_back).
enum Mode {
  kRollout = 0,
  kPolicyRows = 1,
  kValueRows = 2,
  kBackRows = 3,
  kLearnPolicy = 4,
  kLearnValue = 5
};

// Backward image: the W1 slot holds W3^T (rows n < 256, K columns k < out:
// W3[k][n], the rest zero), the W2 slot W2^T (row n, column k: W2[k][n]).
constexpr uint32_t kBackImage = kOffW2 + kW2Bytes;

// -------------------------------------------------------------------------
// weight packing
// -------------------------------------------------------------------------
__device__ __forceinline__ uint16_t bf16_bits(float x) {
  return (uint16_t)(tc::pack_bf16x2(x, 0.0f) & 0xFFFFu);
}

// Column of W1 (and of the observation tile) holding b1's bf16 high part; the
// low part follows.  Above every network input width (<= 18).
constexpr int kBiasCol = 30;

// One thread per 16-byte piece of the W1/W2/W3 regions, then the vectors.
// in_dim: network input width (18 or 12, <= 32); out_dim: 1 (value) or the
// policy head width (<= 16; head rows out_dim..15 are packed as zeros).
__device__ void pack_piece(const float* __restrict__ w, int in_dim, int out_dim,
                           uint8_t* __restrict__ img, int piece) {
  const float* W1 = w;
  const float* b1 = W1 + kH * in_dim;
  const float* W2 = b1 + kH;
  const float* b2 = W2 + kH * kH;
  const float* W3 = b2 + kH;
  const float* b3 = W3 + out_dim * kH;
  const bool policy = out_dim > 1;
  const int n_w1 = kH * 4, n_w2 = 4 * kH * 8, n_w3 = policy ? 4 * kHeadOut * 8 : 0;
  uint16_t v[8];
  uint32_t off;
  if (piece < n_w1) {
    const int n = piece >> 2, p = piece & 3, q = p ^ ((n >> 1) & 3);
    const uint16_t b_hi = bf16_bits(b1[n]);
    const uint16_t b_lo = bf16_bits(b1[n] - __uint_as_float((uint32_t)b_hi << 16));
    for (int e = 0; e < 8; ++e) {
      const int k = 8 * q + e;
      v[e] = k < in_dim ? bf16_bits(W1[n * in_dim + k])
                        : (k == kBiasCol ? b_hi : (k == kBiasCol + 1 ? b_lo : (uint16_t)0));
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
    for (int e = 0; e < 8; ++e)
      v[e] = n < out_dim ? bf16_bits(W3[n * kH + 64 * a + 8 * q + e]) : (uint16_t)0;
    off = kOffW3 + a * (kHeadOut * 128) + n * 128 + p * 16;
  } else {
    const int id = piece - n_w1 - n_w2 - n_w3;   // vector entries, one float each
    float* f = reinterpret_cast<float*>(img);
    if (policy) {
      if (id < kH) f[(kOffB1P >> 2) + id] = b1[id];
      else if (id < 2 * kH) f[(kOffB2P >> 2) + id - kH] = b2[id - kH];
      else if (id < 2 * kH + kHeadOut)
        f[(kOffB3P >> 2) + id - 2 * kH] = id - 2 * kH < out_dim ? b3[id - 2 * kH] : 0.0f;
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

// Backward image of one network from its flat fp32 weights (the layout of
// k_pack): one thread per 16-byte piece of the W1 slot (W3^T, K = 32 with the
// columns from out_dim up zero) and of the W2 slot (W2^T).
__device__ void pack_back_piece(const float* __restrict__ w, int in_dim, int out_dim,
                                uint8_t* __restrict__ img, int piece) {
  const float* W2 = w + kH * in_dim + kH;
  const float* W3 = W2 + kH * kH + kH;
  const int n_w1 = kH * 4, n_w2 = 4 * kH * 8;
  uint16_t v[8];
  uint32_t off;
  if (piece < n_w1) {
    const int n = piece >> 2, p = piece & 3, q = p ^ ((n >> 1) & 3);
    for (int e = 0; e < 8; ++e) {
      const int k = 8 * q + e;
      v[e] = k < out_dim ? bf16_bits(W3[k * kH + n]) : (uint16_t)0;
    }
    off = kOffW1 + n * 64 + p * 16;
  } else if (piece < n_w1 + n_w2) {
    const int id = piece - n_w1;
    const int a = id / (kH * 8), n = (id / 8) % kH, p = id & 7, q = p ^ (n & 7);
    for (int e = 0; e < 8; ++e) v[e] = bf16_bits(W2[(64 * a + 8 * q + e) * kH + n]);
    off = kOffW2 + a * (kH * 128) + n * 128 + p * 16;
  } else {
    return;
  }
  uint4 pk;
  pk.x = v[0] | ((uint32_t)v[1] << 16);
  pk.y = v[2] | ((uint32_t)v[3] << 16);
  pk.z = v[4] | ((uint32_t)v[5] << 16);
  pk.w = v[6] | ((uint32_t)v[7] << 16);
  *reinterpret_cast<uint4*>(img + off) = pk;
}

// Pieces per image (pack_piece: W1, W2, W3 slots, then the vector entries;
// pack_back_piece: W1 and W2 slots).
constexpr int kPolPieces = kH * 4 + 4 * kH * 8 + 4 * kHeadOut * 8 + 2 * kH + kHeadOut;
constexpr int kValPieces = kH * 4 + 4 * kH * 8 + 3 * kH + 1;
constexpr int kBackPieces = kH * 4 + 4 * kH * 8;

__global__ void k_pack(const float* __restrict__ w, int in_dim, int out_dim,
                       uint8_t* __restrict__ img) {
  const int piece = blockIdx.x * blockDim.x + threadIdx.x;
  if (piece < (out_dim > 1 ? kPolPieces : kValPieces)) pack_piece(w, in_dim, out_dim, img, piece);
}

__global__ void k_pack_back(const float* __restrict__ w, int in_dim, int out_dim,
                            uint8_t* __restrict__ img) {
  const int piece = blockIdx.x * blockDim.x + threadIdx.x;
  if (piece < kBackPieces) pack_back_piece(w, in_dim, out_dim, img, piece);
}

// The learner's four images in one launch: blockIdx.y = 0 policy forward,
// 1 value forward, 2 policy backward, 3 value backward (a NULL weight
// pointer skips its images).
struct LearnerImages {
  const float* w[2];   // flat fp32 weights, policy and value
  int in_dim, out_dim[2];
  uint8_t* fwd[2];
  uint8_t* back[2];
};
__global__ void k_pack_learner(const LearnerImages L) {
  const int job = blockIdx.y, net = job & 1;
  const int piece = blockIdx.x * blockDim.x + threadIdx.x;
  if (!L.w[net]) return;
  if (job < 2) {
    if (piece < (net ? kValPieces : kPolPieces)) pack_piece(L.w[net], L.in_dim, L.out_dim[net], L.fwd[net], piece);
  } else if (piece < kBackPieces) {
    pack_back_piece(L.w[net], L.in_dim, L.out_dim[net], L.back[net], piece);
  }
}

// -------------------------------------------------------------------------
// engine
// -------------------------------------------------------------------------
struct Barriers {
  uint64_t obs_full[4];     // group g's observation tile written (128 arrivals)
  uint64_t full_x[4];       // layer-1 chunk 2 or 3 of group g in X (MMA commit)
  uint64_t full_l1a[4];     // layer-1 chunk 0 of group g in its h1 slot, columns 0..63
  uint64_t full_l1b[4];     // layer-1 chunk 1 of group g in its h1 slot, columns 64..127
  uint64_t full_y[4];       // layer-2 even chunk of group g in Y
  uint64_t full_z[4];       // layer-2 odd chunk of group g in Z
  uint64_t acc3_full[4];    // head accumulator of group g complete
  uint64_t empty_x, empty_y, empty_z;   // accumulator read back (128 arrivals)
  uint64_t h1_full[2];      // h1 slot complete (128 arrivals)
  uint64_t h1_part[2][4];   // one group per CTA: h1 chunk c of slot s written (128 arrivals)
  uint64_t h2_part[4];      // one group per CTA: h2 chunk c in tensor memory (both warpgroups)
  uint64_t h2_full[2];      // h2 buffer written (128 arrivals)
  uint64_t acc3_empty[2];   // head slot read back (128 arrivals)
  uint64_t h1_free[2];      // layer-2 MMAs reading an h1 slot completed (commit)
  uint64_t h2_empty[2];     // layer-3 MMAs reading an h2 buffer completed (commit)
  uint64_t drain, drain1, drain2;
  uint64_t img_full;        // the weight image landed (bulk copies, transaction count)
  uint32_t tmem_base;
  int abort;
};

struct RowIO {            // row modes: obs element (r, k) at ((r / ns) * obs_dim + k) * ns + r % ns
  const float* obs;
  size_t rows;
  int ns;
  float* out;             // head[r][out_dim] (policy) or value[r] (value)
  int obs_dim;            // 18 (Fossen model) or 12 (paper model)
  int out_dim;            // policy head width written per row
  // learner rows (zero when unused)
  const uint16_t* xb;     // bf16 inputs xb[r * ldx + k] in place of obs
  int ldx;
  uint16_t* h1;           // bf16 hidden activations h1[r * ldh + j], j < 256
  uint16_t* h2;           // (backward mode: dL/dZ2 and dL/dZ1)
  int ldh;
  int ldo;                // head row stride (0: out_dim for the policy, 1 for the value)
  // backward mode: the forward's H2 and H1 rows a1[r * lda + j], a2[r * lda + j]
  // and the row stride of the second output (0: ldh)
  const uint16_t* a1;
  const uint16_t* a2;
  int lda;
  int ldh2;
  // every learner row (h1, h2, a1, a2; a 16-wide policy head) starts on a
  // 32-byte boundary: rows move as 32-byte pieces, whole L2 sectors
  int wide;
};

// Row pieces as whole 32-byte sectors (sm_100 and later: 256-bit loads and
// stores).  A thread's row piece is otherwise half a sector per access, and
// the warp's 32 rows make 32 partial-sector requests.
__device__ __forceinline__ void st_b32x8(void* p, uint32_t a, uint32_t b, uint32_t c, uint32_t d,
                                         uint32_t e, uint32_t f, uint32_t g, uint32_t h) {
  asm volatile("st.global.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(p), "r"(a),
               "r"(b), "r"(c), "r"(d), "r"(e), "r"(f), "r"(g), "r"(h)
               : "memory");
}

__device__ __forceinline__ void ld_b32x8(const void* p, uint4& lo, uint4& hi) {
  asm volatile("ld.global.nc.v8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
               : "=r"(lo.x), "=r"(lo.y), "=r"(lo.z), "=r"(lo.w), "=r"(hi.x), "=r"(hi.y),
                 "=r"(hi.z), "=r"(hi.w)
               : "l"(p));
}

// 32 bf16 values (64 bytes, 16-byte aligned; wide: 32-byte aligned) from
// global memory.
__device__ __forceinline__ void ld_bf16x32(const uint16_t* h, uint4 (&u)[4], bool wide = false) {
  if (wide) {
    ld_b32x8(h, u[0], u[1]);
    ld_b32x8(h + 16, u[2], u[3]);
    return;
  }
  const uint4* q = reinterpret_cast<const uint4*>(h);
#pragma unroll
  for (int p = 0; p < 4; ++p) u[p] = __ldg(q + p);
}

// Ask for the 128-byte lines of a row of `bytes` bytes to be brought into L2.
__device__ __forceinline__ void prefetch_row_l2(const void* p, int bytes) {
  const char* c = static_cast<const char*>(p);
  for (int o = 0; o < bytes; o += 128) asm volatile("prefetch.global.L2 [%0];" ::"l"(c + o));
  asm volatile("prefetch.global.L2 [%0];" ::"l"(c + bytes - 1));
}

// 32 accumulator columns times tanh' from the forward's bf16 activations h
// (32 values): g (1 - h^2), rounded to 16 bf16 pairs.
__device__ __forceinline__ void dtanh32(const uint32_t (&acc)[32], const uint4 (&hv)[4],
                                        uint32_t (&out)[16]) {
#pragma unroll
  for (int p = 0; p < 4; ++p) {
    const uint4 u = hv[p];
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int j = 4 * p + e;
      const float lo = tc::bf16lo(w[e]), hi = tc::bf16hi(w[e]);
      out[j] = tc::pack_bf16x2(__uint_as_float(acc[2 * j]) * fmaf(-lo, lo, 1.0f),
                               __uint_as_float(acc[2 * j + 1]) * fmaf(-hi, hi, 1.0f));
    }
  }
}

// The same, reading the activations at h (16-byte aligned) when needed.
__device__ __forceinline__ void dtanh32(const uint32_t (&acc)[32], const uint16_t* h,
                                        uint32_t (&out)[16]) {
  uint4 u[4];
  ld_bf16x32(h, u);
  dtanh32(acc, u, out);
}

// 32 bf16 values (16 pairs) to 64 bytes at p (16-byte aligned; wide:
// 32-byte aligned).
__device__ __forceinline__ void store_bf16x32(uint16_t* p, const uint32_t (&v)[16],
                                              bool wide = false) {
  if (wide) {
    st_b32x8(p, v[0], v[1], v[2], v[3], v[4], v[5], v[6], v[7]);
    st_b32x8(p + 16, v[8], v[9], v[10], v[11], v[12], v[13], v[14], v[15]);
    return;
  }
  uint4* q = reinterpret_cast<uint4*>(p);
#pragma unroll
  for (int j = 0; j < 4; ++j) q[j] = make_uint4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
}

template <int G, int MODE>
struct Engine {
  static constexpr bool kPolicy =
      MODE == kRollout || MODE == kPolicyRows || MODE == kLearnPolicy;
  static constexpr bool kBack = MODE == kBackRows;
  static constexpr bool kLearn = MODE >= kBackRows;
  static constexpr uint32_t kImage = kPolicy ? kPolicyImage : (kBack ? kBackImage : kValueImage);
  static constexpr uint32_t kImageAl = (kImage + 1023u) & ~1023u;
  static constexpr uint32_t kOffObs = kImageAl;
  static constexpr uint32_t kOffH2 = kOffObs + G * kObsTileBytes;
  static constexpr uint32_t kOffBar = kOffH2 + (kPolicy ? 2 * kH2TileBytes : 0);
  // The paper model's action history in shared memory (one column per
  // thread, copied in and out once per launch) where it fits: one group.
  static constexpr bool kHistSmem = MODE == kRollout && G == 1;
  static constexpr uint32_t kOffHist = (kOffBar + sizeof(Barriers) + 15u) & ~15u;
  static constexpr uint32_t kHistBytes = kHistSmem ? 6u * paper::kHist * kRows * 4u : 0u;
  static constexpr uint32_t kSmem = kOffHist + kHistBytes + 1024;   // + alignment slack
  static_assert(kSmem <= 227u * 1024u, "shared memory per CTA");
  // One group per CTA in the rollout: a second warpgroup (warps 4-7, the
  // same tensor-memory lanes) takes the second 32-column half of every
  // epilogue chunk, so each sub-partition runs two epilogue warps.
  // With one group a single h1 slot suffices (layer 1 of the next step waits
  // for this step's physics anyway): h1 stays in slot 0, and layer 1's
  // chunks 0 and 1 accumulate in slot 1's columns, so the two warpgroups'
  // packed halves never overwrite accumulator columns the other still reads.
  static constexpr bool kSplit = MODE == kRollout && G == 1;
  static constexpr int kGroupWarps = kSplit ? 8 : 4 * G;
  static constexpr int kThreads = kGroupWarps * 32 + 96;
};

// Row r of the observation tile (bf16, K = 32, 64-byte swizzle): 4 pieces of
// 16 bytes, piece q at position q ^ ((r >> 1) & 3).  Features NOBS..29 are
// zero, 30 and 31 one (the bias columns).
template <int NOBS>
__device__ __forceinline__ void write_obs_row(uint8_t* tile, int r, const float o[NOBS]) {
  static_assert(NOBS % 2 == 0 && NOBS <= kBiasCol, "observation width");
  uint32_t w[16];
#pragma unroll
  for (int j = 0; j < NOBS / 2; ++j) w[j] = tc::pack_bf16x2(o[2 * j], o[2 * j + 1]);
#pragma unroll
  for (int j = NOBS / 2; j < 15; ++j) w[j] = 0u;
  static_assert(kBiasCol == 30, "bias columns are the last word of the row");
  w[15] = tc::pack_bf16x2(1.0f, 1.0f);
  const int sw = (r >> 1) & 3;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    uint4 v = make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
    *reinterpret_cast<uint4*>(tile + r * 64 + ((q ^ sw) << 4)) = v;
  }
}

// 32 accumulator columns (bias included) -> tanh -> 16 bf16 pairs.
__device__ __forceinline__ void tanh32(const uint32_t (&acc)[32], uint32_t (&out)[16]) {
#pragma unroll
  for (int j = 0; j < 16; ++j)
    out[j] = tc::pack_bf16x2(tc::tanh_f32(__uint_as_float(acc[2 * j])),
                             tc::tanh_f32(__uint_as_float(acc[2 * j + 1])));
}

// 32 accumulator columns + bias -> tanh -> 16 bf16 pairs.  The bias is added
// two columns per instruction (packed fp32 add, round to nearest: the same
// sums as scalar adds).  tanh runs on the fp32 sums (tanh.approx.f32, one
// instruction per value) and the results are rounded to a bf16 pair: three
// instructions per pair, where the packed bf16x2 tanh costs a pack plus
// three (two multi-function-unit operations and a merge) on sm_103.
__device__ __forceinline__ void bias_tanh32(const uint32_t (&acc)[32], const float* bias,
                                            uint32_t (&out)[16]) {
#pragma unroll
  for (int j = 0; j < 16; j += 2) {
    const float4 b = *reinterpret_cast<const float4*>(bias + 2 * j);
    const float2 s0 = __fadd2_rn(make_float2(__uint_as_float(acc[2 * j]), __uint_as_float(acc[2 * j + 1])),
                                 make_float2(b.x, b.y));
    const float2 s1 = __fadd2_rn(make_float2(__uint_as_float(acc[2 * j + 2]), __uint_as_float(acc[2 * j + 3])),
                                 make_float2(b.z, b.w));
    out[j] = tc::pack_bf16x2(tc::tanh_f32(s0.x), tc::tanh_f32(s0.y));
    out[j + 1] = tc::pack_bf16x2(tc::tanh_f32(s1.x), tc::tanh_f32(s1.y));
  }
}

// The step's 8 action normals in the tensor-core path's precision class: the
// Philox words and Box-Muller steps of action_noise, with the hardware
// approximations of log and sin/cos (absolute error about 1e-6 on a normal,
// far below the bf16 network's own error on the action it perturbs).
__device__ __forceinline__ void action_noise_approx(uint32_t env, uint32_t seed, uint64_t t_g,
                                                    float eps[8]) {
  const uint32_t lo = (uint32_t)t_g, hi = (uint32_t)(t_g >> 32);
  const uint4 a = philox10(lo, hi, 0u, 0u, env, seed);
  const uint4 b = philox10(lo, hi, 0u, 1u, env, seed);
  const uint32_t w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const float r = sqrtf(-2.0f * __logf(uniform01(w[2 * k])));
    float sn, cs;
    __sincosf(6.28318530717958648f * uniform01(w[2 * k + 1]), &sn, &cs);
    eps[2 * k] = r * cs;
    eps[2 * k + 1] = r * sn;
  }
}

// Group-steps are numbered in the order the MMA warp serves them: iteration
// it of every group that still has work, groups in ascending order (the
// groups with work always form a prefix).  Index of (it, g):
template <int G>
__device__ __forceinline__ int step_index(int it, int g, const int (&iters)[G]) {
  int k = g;
#pragma unroll
  for (int j = 0; j < G; ++j) k += min(it, iters[j]);
  return k;
}

// Register cap: the 4G+3 warps are spread over the SM's four sub-partitions,
// whose 16K-register files each host up to G+1 warps (G = 4: 5 warps x 32
// lanes x 96 registers <= 16384; G = 2: 3 x 32 x 168 <= 16384).
//
// Schedule.  Two group-steps are in flight: while the tensor pipe runs layer 2
// (and layer 3) of group-step k-1, it also runs layer 1 of group-step k, whose
// epilogue fills the other h1 slot (the MMA thread's event loop is described
// at its code).  Accumulator roles are fixed: X holds
// layer-1 chunks, Y and Z the even and odd layer-2 chunks; h1 and the head
// accumulator alternate between two slots by group-step parity.  Every reuse
// of a buffer is ordered either by an "empty" barrier the MMA thread waits on
// or by a commit: an epilogue only starts after a commit that covers every
// MMA issued before it.
// SIM selects the environment model of the fused rollout (0: Fossen,
// 1: the paper model); the row modes ignore it.
template <int G, int MODE, int SIM>
__global__ void __launch_bounds__(Engine<G, MODE>::kThreads) __maxnreg__(G == 4 ? 96 : 168)
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
  constexpr int kGW = E::kGroupWarps;   // MMA-issuing warps: kGW (layer 2), kGW + 1, kGW + 2
  const bool is_mma_warp = warp >= kGW;

  // ---- set-up: barriers, weights, tensor memory ----
  if (tid == 0) {
    for (int g = 0; g < G; ++g) {
      tc::mbar_init(&bar->obs_full[g], kRows);
      tc::mbar_init(&bar->full_x[g], 1);
      tc::mbar_init(&bar->full_l1a[g], 1);
      tc::mbar_init(&bar->full_l1b[g], 1);
      tc::mbar_init(&bar->full_y[g], 1);
      tc::mbar_init(&bar->full_z[g], 1);
      tc::mbar_init(&bar->acc3_full[g], 1);
    }
    // epilogue arrivals: 128, or 256 with the split warpgroups
    constexpr uint32_t kEpi = kRows * (E::kSplit ? 2 : 1);
    tc::mbar_init(&bar->empty_x, kEpi);
    tc::mbar_init(&bar->empty_y, kEpi);
    tc::mbar_init(&bar->empty_z, kEpi);
    for (int s = 0; s < 2; ++s) {
      tc::mbar_init(&bar->h1_full[s], kEpi);
      for (int c = 0; c < kNChunks; ++c) tc::mbar_init(&bar->h1_part[s][c], kEpi);
      if (s == 0)
        for (int c = 0; c < kNChunks; ++c) tc::mbar_init(&bar->h2_part[c], kEpi);
      tc::mbar_init(&bar->h2_full[s], kEpi);
      tc::mbar_init(&bar->acc3_empty[s], kRows);
      tc::mbar_init(&bar->h1_free[s], 1);
      tc::mbar_init(&bar->h2_empty[s], 1);
    }
    tc::mbar_init(&bar->drain, 1);
    tc::mbar_init(&bar->drain1, 1);
    tc::mbar_init(&bar->drain2, 1);
    tc::mbar_init(&bar->img_full, 1);
    bar->abort = 0;
    tc::mbar_fence_init();
    // the weight image in a few bulk copies (16-byte multiples; the image
    // and the shared-memory base are 1024-byte aligned)
    static_assert(E::kImage % 16 == 0, "image size");
    constexpr uint32_t kPiece = 32768;
    tc::mbar_arrive_expect_tx(&bar->img_full, E::kImage);
    for (uint32_t o = 0; o < E::kImage; o += kPiece)
      tc::bulk_g2s(smem + o, image + o, E::kImage - o < kPiece ? E::kImage - o : kPiece,
                   &bar->img_full);
  }
  if (warp == kGW) {
    tc::tmem_alloc(&bar->tmem_base, kTmemCols);
    tc::tmem_relinquish();
  }
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = bar->tmem_base;
  const uint32_t s_base = tc::smem_u32(smem);
  // every role reads the weights (MMA operands, biases): wait for the image
  const bool img_ok = tc::mbar_wait(&bar->img_full, 0, abort, kWaitLimitNs);

  // ---- work assignment ----
  const int n_tiles = MODE == kRollout ? (M.n + kRows - 1) / kRows
                                       : (int)((io.rows + kRows - 1) / kRows);
  const int slot0 = blockIdx.x * G;
  const int n_slots = gridDim.x * G;
  int iters[G];
#pragma unroll
  for (int g = 0; g < G; ++g) {
    const int s = slot0 + g;
    iters[g] = MODE == kRollout ? (s < n_tiles ? T : 0)
                                : (s < n_tiles ? (n_tiles - s - 1) / n_slots + 1 : 0);
    if (!img_ok) iters[g] = 0;   // the wait gave up: no work, the status latches it
  }

  if (is_mma_warp) {
    // =================== MMA issue: three streams, one elected lane each ===================
    // Warp 4G+1 issues layer 1 of each group-step into X chunk by chunk;
    // warp 4G issues layer 2 (chunks c0..c3 into Y, Z, Y, Z) once the step's
    // h1 is complete; warp 4G+2 issues layer 3 chunk by chunk as the h2
    // buffers fill (policy modes).  Each thread blocks (suspended by the
    // hardware) only on the barrier of its own next operation, so no stream
    // waits behind another's epilogue: layer 2 of step k+1 starts as soon as
    // its h1 and an accumulator are ready, while layer 3 of step k is still
    // waiting for step k's last h2 chunk.  Before layer 1 of step k the
    // layer-1 thread waits until the layer-2 MMAs of step k-2, which read the
    // same h1 slot, have completed (h1_free).
    if ((tid & 31) == 0) {
      constexpr uint32_t kI64 = tc::idesc_bf16_f32(128, kChunk);
      constexpr uint32_t kI16 = tc::idesc_bf16_f32(128, kHeadOut);
      int total = 0;
#pragma unroll
      for (int g = 0; g < G; ++g) total += iters[g];
      // iters[] is read with a runtime index through selects, so that it stays
      // in registers (likewise the per-slot barrier phases below are bits).
      auto iters_at = [&](int gg) {
        int v = 0;
#pragma unroll
        for (int j = 0; j < G; ++j) v = j == gg ? iters[j] : v;
        return v;
      };
      auto advance = [&](int& it, int& g) {
        ++g;
        if (g >= G || iters_at(g) <= it) {
          g = 0;
          ++it;
        }
      };
      bool ok = true;
      int it = 0, g = 0;
      // One group per CTA: no other group's layer 2 fills the tensor pipe
      // while this group's layer-1 epilogue runs, so layer 2's chunks 0 and
      // 1 (accumulators Y and Z, both drained by then) are fed K-slice by
      // K-slice as h1's chunks are written (h1_part), not after all of h1.
      constexpr bool kProgL2 = G == 1 && MODE == kRollout;
      if (warp == kGW) {
        uint32_t u_y = 0, u_z = 0;
        uint32_t p_h1 = 0;   // phase bit of slot s at bit s
        auto issue_l2 = [&](int k, int g2, int c) -> bool {
          const int s2 = E::kSplit ? 0 : k & 1;
          const bool odd = c & 1;
          uint32_t& u = odd ? u_z : u_y;
          const bool r = tc::mbar_wait(odd ? &bar->empty_z : &bar->empty_y, (u & 1u) ^ 1u, abort,
                                       kWaitLimitNs);
          ++u;
          if (!r) return false;
          tc::tc_fence_after();
          const uint32_t d = tmem + (odd ? kColZ : kColY);
          const uint32_t a0 = tmem + kColH1 + s2 * 128;
          // descriptor start addresses are in 16-byte units: step K by adding offsets
          const uint64_t b0 = tc::smem_desc(s_base + kOffW2 + c * kChunk * 128, 1024, 2);
#pragma unroll
          for (int kk = 0; kk < 16; ++kk)
            tc::mma_ts(d, a0 + kk * 8, b0 + (uint64_t)(((kk >> 2) * (kH * 128) + (kk & 3) * 32) >> 4),
                       kI64, kk > 0 ? 1u : 0u);
          tc::mma_commit(odd ? &bar->full_z[g2] : &bar->full_y[g2]);
          if (c == kNChunks - 1) tc::mma_commit(&bar->h1_free[s2]);
          return true;
        };
        for (int k = 0; k < total && ok; ++k) {
          const int s2 = E::kSplit ? 0 : k & 1;
          if constexpr (kProgL2) {
            // chunks 0 and 1 (Y, Z) K-slice by K-slice as h1's chunks land
            ok = tc::mbar_wait(&bar->empty_y, (u_y & 1u) ^ 1u, abort, kWaitLimitNs) &&
                 tc::mbar_wait(&bar->empty_z, (u_z & 1u) ^ 1u, abort, kWaitLimitNs);
            ++u_y;
            ++u_z;
            const uint32_t a0 = tmem + kColH1 + s2 * 128;
            const uint64_t by = tc::smem_desc(s_base + kOffW2, 1024, 2);
            const uint64_t bz = tc::smem_desc(s_base + kOffW2 + kChunk * 128, 1024, 2);
            for (int c = 0; c < kNChunks && ok; ++c) {
              ok = tc::mbar_wait(&bar->h1_part[s2][c], (p_h1 >> s2) & 1u, abort, kWaitLimitNs);
              if (!ok) break;
              tc::tc_fence_after();
#pragma unroll
              for (int q = 0; q < 4; ++q) {
                const int kk = 4 * c + q;
                const uint64_t off = (uint64_t)(((kk >> 2) * (kH * 128) + (kk & 3) * 32) >> 4);
                tc::mma_ts(tmem + kColY, a0 + kk * 8, by + off, kI64, kk > 0 ? 1u : 0u);
                tc::mma_ts(tmem + kColZ, a0 + kk * 8, bz + off, kI64, kk > 0 ? 1u : 0u);
              }
            }
            p_h1 ^= 1u << s2;
            if (!ok) break;
            tc::mma_commit(&bar->full_y[g]);
            tc::mma_commit(&bar->full_z[g]);
            ok = issue_l2(k, g, 2) && issue_l2(k, g, 3);
          } else {
            ok = tc::mbar_wait(&bar->h1_full[s2], (p_h1 >> s2) & 1u, abort, kWaitLimitNs);
            p_h1 ^= 1u << s2;
            if (!ok) break;
            tc::tc_fence_after();
            ok = issue_l2(k, g, 0) && issue_l2(k, g, 1) && issue_l2(k, g, 2) && issue_l2(k, g, 3);
          }
          advance(it, g);
        }
      } else if (warp == kGW + 2) {
        // layer 3: A = h2 buffer (c & 1), B = W3 K-slice c, into head slot k & 1
        uint32_t p_h2 = 0, p_a3 = 0;   // phase bit of buffer / slot s at bit s
        for (int k = 0; k < total && ok && kPolicy; ++k) {
          const int s2 = k & 1;
          ok = tc::mbar_wait(&bar->acc3_empty[s2], ((p_a3 >> s2) & 1u) ^ 1u, abort, kWaitLimitNs);
          p_a3 ^= 1u << s2;
          for (int c = 0; c < kNChunks && ok; ++c) {
            if constexpr (E::kSplit) {
              // h2 chunk c in tensor memory (columns 128 + 32c.., packed bf16)
              ok = tc::mbar_wait(&bar->h2_part[c], (uint32_t)k & 1u, abort, kWaitLimitNs);
              if (!ok) break;
              tc::tc_fence_after();
              const uint32_t a0 = tmem + kColH1 + 128 + c * 32;
              const uint64_t b0 = tc::smem_desc(s_base + kOffW3 + c * (kHeadOut * 128), 1024, 2);
#pragma unroll
              for (int kk = 0; kk < 4; ++kk)
                tc::mma_ts(tmem + kColA3 + s2 * 16, a0 + kk * 8, b0 + (uint64_t)(kk * 2), kI16,
                           (c > 0 || kk > 0) ? 1u : 0u);
              if (c == kNChunks - 1) tc::mma_commit(&bar->acc3_full[g]);
              continue;
            }
            const int hb = c & 1;
            ok = tc::mbar_wait(&bar->h2_full[hb], (p_h2 >> hb) & 1u, abort, kWaitLimitNs);
            p_h2 ^= 1u << hb;
            if (!ok) break;
            tc::tc_fence_after();
            const uint64_t a0 = tc::smem_desc(s_base + E::kOffH2 + hb * kH2TileBytes, 1024, 2);
            const uint64_t b0 = tc::smem_desc(s_base + kOffW3 + c * (kHeadOut * 128), 1024, 2);
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              tc::mma_ss(tmem + kColA3 + s2 * 16, a0 + (uint64_t)(kk * 2), b0 + (uint64_t)(kk * 2),
                         kI16, (c > 0 || kk > 0) ? 1u : 0u);
            tc::mma_commit(&bar->h2_empty[hb]);
            if (c == kNChunks - 1) tc::mma_commit(&bar->acc3_full[g]);
          }
          advance(it, g);
        }
      } else {
        uint32_t u_x = 0, p_hf = 0, p_obs = 0;   // phase bits per slot / group
        for (int k = 0; k < total && ok; ++k) {
          const int s1 = E::kSplit ? 0 : k & 1;
          ok = tc::mbar_wait(&bar->h1_free[s1], ((p_hf >> s1) & 1u) ^ 1u, abort, kWaitLimitNs);
          p_hf ^= 1u << s1;
          if (!ok) break;
          ok = tc::mbar_wait(&bar->obs_full[g], (p_obs >> g) & 1u, abort, kWaitLimitNs);
          p_obs ^= 1u << g;
          const uint32_t obs_s = s_base + E::kOffObs + g * kObsTileBytes;
          // Chunks 0 and 1 accumulate in the step's own h1 slot (free since
          // h1_free; the epilogue overwrites it with the bf16 h1 only where
          // it has read the accumulator), chunks 2 and 3 in X.  So three
          // chunks start at once and only chunk 3 waits for X to drain.
          for (int c = 0; c < kNChunks && ok; ++c) {
            uint32_t d = tmem + kColH1 + (E::kSplit ? 128 : s1 * 128) + c * kChunk;
            if (c >= 2) {
              ok = tc::mbar_wait(&bar->empty_x, (u_x & 1u) ^ 1u, abort, kWaitLimitNs);
              ++u_x;
              if (!ok) break;
              d = tmem + kColX;
            }
            tc::tc_fence_after();
            const uint64_t a0 = tc::smem_desc(obs_s, 512, 4);
            const uint64_t b0 = tc::smem_desc(s_base + kOffW1 + c * kChunk * 64, 512, 4);
            tc::mma_ss(d, a0, b0, kI64, 0u);
            tc::mma_ss(d, a0 + 2, b0 + 2, kI64, 1u);
            tc::mma_commit(c == 0 ? &bar->full_l1a[g] : (c == 1 ? &bar->full_l1b[g] : &bar->full_x[g]));
          }
          advance(it, g);
        }
      }
      // drain: every MMA this thread issued has completed before tensor memory is freed
      uint64_t* drain = warp == kGW ? &bar->drain : (warp == kGW + 1 ? &bar->drain1 : &bar->drain2);
      tc::mma_commit(drain);
      tc::mbar_wait(drain, 0, abort, kWaitLimitNs);
    }
    __syncwarp();
  } else {
    // =================== groups: epilogues + physics / row I/O ===================
    const int g = E::kSplit ? 0 : warp >> 2;
    const int row = tid & (kRows - 1);
    // split epilogues: warps 0-3 take the first 32 columns of every chunk
    // (and the head, sampling and physics), warps 4-7 the second
    const bool helper = E::kSplit && warp >= 4;
    const int half_lo = E::kSplit ? (helper ? 1 : 0) : 0;
    const int half_hi = E::kSplit ? half_lo + 1 : 2;
    const uint32_t lane_addr = tmem + ((uint32_t)((warp & 3) * 32) << 16);
    uint8_t* obs_tile = smem + E::kOffObs + g * kObsTileBytes;
    uint8_t* h2_tiles = smem + E::kOffH2;
    const float* b2 = reinterpret_cast<const float*>(smem + (kPolicy ? kOffB2P : kOffB2V));
    // Barrier phases need no counters: per group-step a group waits on its
    // full_x, full_y and full_z barriers twice each and on full_l1a,
    // full_l1b and acc3_full once, so the phase parities are c & 1,
    // (c >> 1) & 1 and the parity of the group's own step count.
    bool ok = true;

    // Layer 1-3 epilogues of this group's step k; value mode returns the
    // head dot product in head[0], policy mode the 16 head outputs.  With
    // h1r / h2r set, the row's bf16 hidden activations are stored there too.
    auto run_network = [&](int k, int it, float* head, uint16_t* h1r, uint16_t* h2r,
                           const uint16_t* a1r, const uint16_t* a2r) -> bool {
      const int slot = E::kSplit ? 0 : k & 1;
      // Backward with at most two groups (registers to spare): the forward
      // activations tanh' needs are loaded one chunk ahead of their use, so
      // that their memory latency overlaps the tensor-core work instead of
      // sitting between an accumulator read and its epilogue.
      constexpr bool kPreA = E::kBack && G <= 2;
      uint4 pa[2][4];
      const bool wide = io.wide != 0;
      if constexpr (kPreA) {
        ld_bf16x32(a1r, pa[0], wide);
        ld_bf16x32(a1r + 32, pa[1], wide);
      }
      // layer 1 -> h1 slot.  Chunk c's bf16 pairs go to slot columns
      // 32c..32c+31, which held accumulator columns this thread has already
      // read (chunk 0's second half for c = 1, chunk 1's for c = 2, 3).
      // The Fossen rollout keeps this loop rolled: its hot loop (network
      // epilogues, sampling, physics) otherwise outgrows the SM's instruction
      // cache, and with every SM busy the misses cost more than the loop
      // (2.52 -> 2.19 ms at 152 CTAs, 2.02 -> 1.95 ms at 128).  The paper
      // model and the row modes run faster unrolled.
#pragma unroll(MODE == kRollout && SIM == 0 ? 1 : 4)
      for (int c = 0; c < kNChunks; ++c) {
        uint64_t* full = c == 0 ? &bar->full_l1a[g] : (c == 1 ? &bar->full_l1b[g] : &bar->full_x[g]);
        if (!tc::mbar_wait(full, c < 2 ? (uint32_t)it & 1u : (uint32_t)c & 1u, abort, kWaitLimitNs))
          return false;
        tc::tc_fence_after();
        const uint32_t src =
            c < 2 ? kColH1 + (E::kSplit ? 128 : slot * 128) + c * kChunk : kColX;
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          if (E::kSplit && (half < half_lo || half >= half_hi)) continue;
          uint32_t acc[32], hv[16];
          tc::tmem_ld32(lane_addr + src + 32 * half, acc);
          tc::tmem_ld_wait(acc);
          if ((E::kSplit || half == 1) && c >= 2) {
            tc::tc_fence_before();
            tc::mbar_arrive(&bar->empty_x);
          }
          if constexpr (kPreA) {
            uint4 cur[4];
#pragma unroll
            for (int p = 0; p < 4; ++p) cur[p] = pa[half][p];
            // next: this half of chunk c + 1, or of layer 2's chunk 0
            ld_bf16x32(c + 1 < kNChunks ? a1r + (c + 1) * kChunk + 32 * half : a2r + 32 * half,
                       pa[half], wide);
            dtanh32(acc, cur, hv);
          } else if constexpr (E::kBack) {
            dtanh32(acc, a1r + c * kChunk + 32 * half, hv);
          } else {
            tanh32(acc, hv);
          }
          tc::tmem_st16(lane_addr + kColH1 + slot * 128 + c * 32 + half * 16, hv);
          if (E::kLearn && h1r) store_bf16x32(h1r + c * kChunk + 32 * half, hv, wide);
        }
        if constexpr (G == 1 && MODE == kRollout) {   // chunk c announced (layer 2 starts on it)
          tc::tmem_st_wait();
          tc::tc_fence_before();
          tc::mbar_arrive(&bar->h1_part[slot][c]);
        }
      }
      if constexpr (!(G == 1 && MODE == kRollout)) {
        tc::tmem_st_wait();
        tc::tc_fence_before();
        tc::mbar_arrive(&bar->h1_full[slot]);
      }
      float2 vsum = make_float2(0.0f, 0.0f);   // value head: even and odd columns
      const float* w3v = reinterpret_cast<const float*>(smem + kOffW3V);
      for (int c = 0; c < kNChunks; ++c) {       // layer 2 (Y / Z)
        const bool odd = c & 1;
        if (!tc::mbar_wait(odd ? &bar->full_z[g] : &bar->full_y[g], ((uint32_t)c >> 1) & 1u, abort,
                           kWaitLimitNs))
          return false;
        tc::tc_fence_after();
        const uint32_t col = odd ? kColZ : kColY;
        uint8_t* h2 = h2_tiles + (c & 1) * kH2TileBytes + row * 128;
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          if (E::kSplit && (half < half_lo || half >= half_hi)) continue;
          uint32_t acc[32], hv[16];
          tc::tmem_ld32(lane_addr + col + 32 * half, acc);
          tc::tmem_ld_wait(acc);
          if (E::kSplit || half == 1) {
            tc::tc_fence_before();
            tc::mbar_arrive(odd ? &bar->empty_z : &bar->empty_y);
          }
          if constexpr (kPreA) {
            uint4 cur[4];
#pragma unroll
            for (int p = 0; p < 4; ++p) cur[p] = pa[half][p];
            if (c + 1 < kNChunks) ld_bf16x32(a2r + (c + 1) * kChunk + 32 * half, pa[half], wide);
            dtanh32(acc, cur, hv);
          } else if constexpr (E::kBack) {
            dtanh32(acc, a2r + c * kChunk + 32 * half, hv);
          } else {
            bias_tanh32(acc, b2 + c * kChunk + 32 * half, hv);
          }
          if (E::kLearn && h2r) store_bf16x32(h2r + c * kChunk + 32 * half, hv, wide);
          if constexpr (E::kBack) {
            // backward: dL/dZ1 goes to global memory only
          } else if (E::kSplit) {
            // one group: h2 stays in tensor memory (columns 128..255, free
            // once layer 1's epilogue has read its accumulators) as layer 3's
            // A operand
            tc::tmem_st16(lane_addr + kColH1 + 128 + c * 32 + half * 16, hv);
          } else if (kPolicy) {
            // Write j = 2k + (c >> 1) of h2 buffer c & 1 reuses it after
            // layer 3 has consumed write j - 1 (completion j - 1 of h2_empty).
            const int j = 2 * k + (c >> 1);
            if (half == 0 && j > 0 &&
                !tc::mbar_wait(&bar->h2_empty[c & 1], (uint32_t)(j - 1) & 1u, abort, kWaitLimitNs))
              return false;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const int pos = (4 * half + q) ^ (row & 7);
              *reinterpret_cast<uint4*>(h2 + (pos << 4)) =
                  make_uint4(hv[4 * q], hv[4 * q + 1], hv[4 * q + 2], hv[4 * q + 3]);
            }
          } else {
            const float4* w = reinterpret_cast<const float4*>(w3v + c * kChunk + 32 * half);
#pragma unroll
            for (int j = 0; j < 16; j += 2) {
              const float4 wv = w[j >> 1];
              vsum = __ffma2_rn(make_float2(tc::bf16lo(hv[j]), tc::bf16hi(hv[j])),
                                make_float2(wv.x, wv.y), vsum);
              vsum = __ffma2_rn(make_float2(tc::bf16lo(hv[j + 1]), tc::bf16hi(hv[j + 1])),
                                make_float2(wv.z, wv.w), vsum);
            }
          }
        }
        if constexpr (E::kSplit) {
          tc::tmem_st_wait();
          tc::tc_fence_before();
          tc::mbar_arrive(&bar->h2_part[c]);
        } else if (kPolicy) {
          tc::fence_async_smem();
          tc::mbar_arrive(&bar->h2_full[c & 1]);
        }
      }
      if constexpr (E::kBack) return true;
      if (!kPolicy) {
        head[0] = (vsum.x + vsum.y) + *reinterpret_cast<const float*>(smem + kOffB3V);
        return true;
      }
      if (helper) return true;   // the head belongs to the first warpgroup
      if (!tc::mbar_wait(&bar->acc3_full[g], (uint32_t)it & 1u, abort, kWaitLimitNs)) return false;
      tc::tc_fence_after();
      uint32_t o3[16];
      // head slot: by group-step parity (layer 3 alternates), also with one
      // h1 slot
      tc::tmem_ld16(lane_addr + kColA3 + (k & 1) * 16, o3);
      tc::tmem_ld_wait(o3);
      tc::tc_fence_before();
      tc::mbar_arrive(&bar->acc3_empty[k & 1]);
      const float* b3 = reinterpret_cast<const float*>(smem + kOffB3P);
#pragma unroll
      for (int j = 0; j < kHeadOut; ++j) head[j] = __uint_as_float(o3[j]) + b3[j];
      return true;
    };

    int my_iters = 0;
#pragma unroll
    for (int j = 0; j < G; ++j) my_iters = j == g ? iters[j] : my_iters;
    if (helper) {
      // the second epilogue warpgroup: the networks only, one item per step
      for (int t = 0; t < my_iters && ok; ++t) {
        float head[kHeadOut];
        ok = run_network(t, t, head, nullptr, nullptr, nullptr, nullptr);
      }
    } else if constexpr (MODE == kRollout && SIM == 0) {
      int n_act = 0;
#pragma unroll
      for (int j = 0; j < G; ++j) n_act += iters[j] > 0 ? 1 : 0;
      const int tile = slot0 + g;
      const int i = tile * kRows + row;
      const bool active = my_iters > 0 && i < M.n;
      const size_t n = (size_t)M.n;
      Env e;
      if (active) load_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
      bool bad = false;
      for (int t = 0; t < my_iters && ok; ++t) {
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
        write_obs_row<kObs>(obs_tile, row, o);
        tc::fence_async_smem();
        tc::mbar_arrive(&bar->obs_full[g]);
        float head[kHeadOut];
        __syncwarp();
        // every group with work runs T steps: the step index is t * n_act + g
        if (!(ok = run_network(t * n_act + g, t, head, nullptr, nullptr, nullptr, nullptr))) break;
        __syncwarp();
        if (active) {
          // The episode parameters are not held in registers across the
          // network (they would not fit beside the accumulators).
          reload_params(M, B.params, i, e);
          const uint32_t id = M.id_base + (uint32_t)i;
          float eps[kAct];
          action_noise_approx(id, M.seed, t_g0 + (uint64_t)t, eps);
          float a[kAct], lp = 0.0f;
#pragma unroll
          for (int k = 0; k < kAct; ++k) {
            const float ls = fminf(fmaxf(head[kAct + k], M.logstd_min), M.logstd_max);
            a[k] = fmaf(__expf(ls), eps[k], head[k]);
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
          if (d) store_params(M, B.params, i, e);
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
    } else if constexpr (MODE == kRollout && SIM == 1) {
      // The paper's own environment: 12-float observation, 6-D wrench
      // action (mean head[0..5], clamped log-std head[6..11]), history in
      // the state rows.
      constexpr int kPO = paper::kObs, kPA = paper::kAct;
      int n_act = 0;
#pragma unroll
      for (int j = 0; j < G; ++j) n_act += iters[j] > 0 ? 1 : 0;
      const int tile = slot0 + g;
      const int i = tile * kRows + row;
      const bool active = my_iters > 0 && i < M.n;
      const size_t n = (size_t)M.n;
      paper::Env e;
      if (active) paper::load_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
      bool bad = false;
      // history rows: global (read past L1), or with one group this thread's
      // shared-memory column
      float* const hist_col = reinterpret_cast<float*>(smem + E::kOffHist) + row;
      if constexpr (E::kHistSmem) {
        if (active) {
          const paper::HistG hg = paper::hist_rows(B.state, M.n, i);
          for (int r = 0; r < 6 * paper::kHist; ++r) hist_col[r * kRows] = hg.ld(r);
        }
      }
      for (int t = 0; t < my_iters && ok; ++t) {
        float o[kPO];
        if (active) {
          paper::observe(e, o);
          if (tr.obs) {
#pragma unroll
            for (int k = 0; k < kPO; ++k) tr.obs[((size_t)t * kPO + k) * n + i] = o[k];
          }
        } else {
#pragma unroll
          for (int k = 0; k < kPO; ++k) o[k] = 0.0f;
        }
        write_obs_row<kPO>(obs_tile, row, o);
        tc::fence_async_smem();
        tc::mbar_arrive(&bar->obs_full[g]);
        float head[kHeadOut];
        // The step's normals depend only on (env, seed, step): with one group
        // per CTA (registers to spare) they are drawn while layer 1 runs
        // instead of after the network.
        constexpr bool kEarlyNoise = G == 1;
        float eps[8];
        if (kEarlyNoise && active) action_noise_approx(M.id_base + (uint32_t)i, M.seed, t_g0 + (uint64_t)t, eps);
        __syncwarp();
        if (!(ok = run_network(t * n_act + g, t, head, nullptr, nullptr, nullptr, nullptr))) break;
        __syncwarp();
        if (active) {
          const uint32_t id = M.id_base + (uint32_t)i;
          if (!kEarlyNoise) action_noise_approx(id, M.seed, t_g0 + (uint64_t)t, eps);
          float a[kPA], lp = 0.0f;
#pragma unroll
          for (int k = 0; k < kPA; ++k) {
            const float ls = fminf(fmaxf(head[kPA + k], M.logstd_min), M.logstd_max);
            a[k] = fmaf(__expf(ls), eps[k], head[k]);
            lp += -0.5f * eps[k] * eps[k] - ls;
          }
          lp -= (float)kPA * 0.91893853320467274f;
          if (tr.act) {
#pragma unroll
            for (int k = 0; k < kPA; ++k) tr.act[((size_t)t * kPA + k) * n + i] = a[k];
          }
          if (tr.logp) tr.logp[(size_t)t * n + i] = lp;
          bool d;
          float r;
          if constexpr (E::kHistSmem)
            r = paper::physics_step(M, id, e, a, paper::HistS{hist_col, kRows}, &d);
          else
            r = paper::physics_step(M, id, e, a, paper::hist_rows(B.state, M.n, i), &d);
          if (tr.rew) tr.rew[(size_t)t * n + i] = r;
          if (tr.done) tr.done[(size_t)t * n + i] = d ? 1 : 0;
          bad |= !paper::env_finite(e);
        }
        __syncwarp();
      }
      if (active) {
        if (bad) flag_nan(st, i);
        paper::store_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
        if constexpr (E::kHistSmem) {
          const paper::HistG hg = paper::hist_rows(B.state, M.n, i);
          for (int r = 0; r < 6 * paper::kHist; ++r) hg.st(r, hist_col[r * kRows]);
        }
      }
    } else {
      // Learner modes with at most two groups: the next iteration's input
      // row is loaded while this one runs (and, backward, the next rows of
      // forward activations are requested into L2), so no iteration starts
      // with a wait on memory.
      constexpr bool kPreX = E::kLearn && G <= 2;
      constexpr int kXq = (kObs + 7) / 8;
      auto load_x = [&](size_t rr, uint4 (&u)[kXq]) {
        const uint4* x = reinterpret_cast<const uint4*>(io.xb + rr * (size_t)io.ldx);
#pragma unroll
        for (int q = 0; q < kXq; ++q)
          u[q] = (rr < io.rows && 8 * q < io.obs_dim) ? __ldg(x + q) : make_uint4(0u, 0u, 0u, 0u);
      };
      uint4 xn[kXq];
      if constexpr (kPreX) load_x((size_t)(slot0 + g) * kRows + row, xn);
      for (int it = 0; it < my_iters && ok; ++it) {
        const size_t r = (size_t)(slot0 + g + it * n_slots) * kRows + row;
        const bool active = r < io.rows;
        float o[kObs];
        uint4 xc[kXq];
        if constexpr (kPreX) {
          const size_t rn = r + (size_t)n_slots * kRows;
#pragma unroll
          for (int q = 0; q < kXq; ++q) xc[q] = xn[q];
          if (it + 1 < my_iters) {
            load_x(rn, xn);
            if (E::kBack && rn < io.rows) {
              prefetch_row_l2(io.a1 + rn * (size_t)io.lda, 2 * kH);
              prefetch_row_l2(io.a2 + rn * (size_t)io.lda, 2 * kH);
            }
          }
        } else if (E::kLearn && active) {
          load_x(r, xc);
        }
        if (E::kLearn && active) {
          // bf16 row, 16-byte pieces (ldx a multiple of 8, >= obs_dim)
#pragma unroll
          for (int q = 0; q < kXq; ++q) {
            const uint4 u = xc[q];
            const uint32_t w4[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              const int k = 8 * q + j;
              if (k < kObs) {
                const float v = (j & 1) ? tc::bf16hi(w4[j >> 1]) : tc::bf16lo(w4[j >> 1]);
                o[k] = k < io.obs_dim ? v : 0.0f;
              }
            }
          }
        } else if (active) {
          const size_t ns = (size_t)io.ns;
          const size_t base = (r / ns) * (size_t)io.obs_dim * ns + r % ns;
#pragma unroll
          for (int k = 0; k < kObs; ++k)
            o[k] = k < io.obs_dim ? __ldg(io.obs + base + (size_t)k * ns) : 0.0f;
        } else {
#pragma unroll
          for (int k = 0; k < kObs; ++k) o[k] = 0.0f;
        }
        write_obs_row<kObs>(obs_tile, row, o);
        tc::fence_async_smem();
        tc::mbar_arrive(&bar->obs_full[g]);
        float head[kHeadOut];
        __syncwarp();
        uint16_t* h1r = E::kLearn && active && io.h1 ? io.h1 + r * (size_t)io.ldh : nullptr;
        uint16_t* h2r = E::kLearn && active && io.h2
                            ? io.h2 + r * (size_t)(io.ldh2 ? io.ldh2 : io.ldh)
                            : nullptr;
        // backward mode: inactive rows read row 0's activations (results unused)
        const size_t ra = active ? r : 0;
        const uint16_t* a1r = E::kBack ? io.a1 + ra * (size_t)io.lda : nullptr;
        const uint16_t* a2r = E::kBack ? io.a2 + ra * (size_t)io.lda : nullptr;
        if (!(ok = run_network(step_index<G>(it, g, iters), it, head, h1r, h2r, a1r, a2r))) break;
        __syncwarp();
        if (active && !E::kBack) {
          if (!E::kPolicy) {
            io.out[r * (size_t)(io.ldo ? io.ldo : 1)] = head[0];
          } else {
            const size_t ldo = (size_t)(io.ldo ? io.ldo : io.out_dim);
            if (E::kLearn && io.wide && io.out_dim == kHeadOut) {
              float* o16 = io.out + r * ldo;
              st_b32x8(o16, __float_as_uint(head[0]), __float_as_uint(head[1]),
                       __float_as_uint(head[2]), __float_as_uint(head[3]), __float_as_uint(head[4]),
                       __float_as_uint(head[5]), __float_as_uint(head[6]), __float_as_uint(head[7]));
              st_b32x8(o16 + 8, __float_as_uint(head[8]), __float_as_uint(head[9]),
                       __float_as_uint(head[10]), __float_as_uint(head[11]),
                       __float_as_uint(head[12]), __float_as_uint(head[13]),
                       __float_as_uint(head[14]), __float_as_uint(head[15]));
            } else {
#pragma unroll
              for (int k = 0; k < kHeadOut; ++k)
                if (k < io.out_dim) io.out[r * ldo + k] = head[k];
            }
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
  if (warp == kGW) {
    tc::tc_fence_after();
    tc::tmem_dealloc(tmem, kTmemCols);
  }
}

// SM count of the current device, looked up once per device (the grids are
// sized per launch for the device the launch goes to).
int sm_count() {
  constexpr int kMaxDev = 64;
  static std::atomic<int> cached[kMaxDev];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) {
    cudaGetLastError();
    dev = 0;
  }
  int v = dev < kMaxDev ? cached[dev].load(std::memory_order_relaxed) : 0;
  if (v <= 0) {
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v <= 0) {
      cudaGetLastError();
      v = 1;
    }
    if (dev < kMaxDev) cached[dev].store(v, std::memory_order_relaxed);
  }
  return v;
}

template <int G, int MODE, int SIM = 0>
cudaError_t launch_engine(int grid, const Model& M, const Buffers& B, const uint8_t* image,
                          const Traj& tr, int T, uint64_t t_g0, const RowIO& io, Status* st,
                          cudaStream_t s) {
  using E = Engine<G, MODE>;
  cudaError_t err = cudaFuncSetAttribute(k_engine<G, MODE, SIM>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, E::kSmem);
  if (err != cudaSuccess) return err;
  k_engine<G, MODE, SIM><<<grid, E::kThreads, E::kSmem, s>>>(M, B, image, tr, T, t_g0, io, st);
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

// Failure-detection self-test: one thread waits, with the engine's bounded
// wait, on a barrier phase that nothing completes; the wait gives up after
// `limit_ns` and the timeout is latched in the status block exactly as an
// engine wait would latch it.
__global__ void k_wait_selftest(Status* st, uint64_t limit_ns) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    tc::mbar_init(&bar, 1);
    abort_flag = 0;
    tc::mbar_fence_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    volatile int* abort = &abort_flag;
    if (!tc::mbar_wait(&bar, 0, abort, limit_ns)) {
      atomicAdd(&st->timeouts, 1);
      atomicCAS(&st->code, 0, -4);
    }
  }
}

}  // namespace

cudaError_t launch_wait_selftest(Status* st, uint64_t limit_ns, cudaStream_t s) {
  k_wait_selftest<<<1, 32, 0, s>>>(st, limit_ns);
  return cudaGetLastError();
}

int engine_sm_count() { return sm_count(); }

size_t bf16_policy_image_bytes() { return kPolicyImage; }
size_t bf16_value_image_bytes() { return kValueImage; }
size_t bf16_back_image_bytes() { return kBackImage; }

cudaError_t launch_pack_back_bf16(int in_dim, int out_dim, const float* w_f32, void* packed,
                                  cudaStream_t s) {
  k_pack_back<<<(kBackPieces + 255) / 256, 256, 0, s>>>(w_f32, in_dim, out_dim,
                                                        static_cast<uint8_t*>(packed));
  return cudaGetLastError();
}

cudaError_t launch_pack_learner_bf16(int in_dim, int policy_out, const float* wp_f32,
                                     const float* wv_f32, void* wp_packed, void* wv_packed,
                                     void* bp_packed, void* bv_packed, cudaStream_t s) {
  const LearnerImages L = {{wp_f32, wv_f32},
                           in_dim,
                           {policy_out, 1},
                           {static_cast<uint8_t*>(wp_packed), static_cast<uint8_t*>(wv_packed)},
                           {static_cast<uint8_t*>(bp_packed), static_cast<uint8_t*>(bv_packed)}};
  constexpr int kMax = kPolPieces > kBackPieces ? kPolPieces : kBackPieces;
  k_pack_learner<<<dim3((kMax + 255) / 256, 4), 256, 0, s>>>(L);
  return cudaGetLastError();
}

cudaError_t launch_pack_bf16(const Model& M, const float* wp_f32, const float* wv_f32,
                             void* wp_packed, void* wv_packed, cudaStream_t s) {
  return launch_pack_bf16_dims(M.model == 1 ? 12 : kObs, M.policy_out, wp_f32, wv_f32, wp_packed,
                               wv_packed, s);
}

cudaError_t launch_pack_bf16_dims(int in_dim, int policy_out, const float* wp_f32,
                                  const float* wv_f32, void* wp_packed, void* wv_packed,
                                  cudaStream_t s) {
  cudaError_t e = cudaSuccess;
  if (wp_f32) {
    k_pack<<<(kPolPieces + 255) / 256, 256, 0, s>>>(wp_f32, in_dim, policy_out,
                                                    static_cast<uint8_t*>(wp_packed));
    e = cudaGetLastError();
  }
  if (e != cudaSuccess || !wv_f32) return e;
  k_pack<<<(kValPieces + 255) / 256, 256, 0, s>>>(wv_f32, in_dim, 1,
                                                  static_cast<uint8_t*>(wv_packed));
  return cudaGetLastError();
}

cudaError_t launch_rollout_bf16(const Model& M, const Buffers& B, const void* wp_packed,
                                const Traj& tr, int T, uint64_t t_g0, Status* st, cudaStream_t s) {
  const long tiles = (M.n + kRows - 1) / kRows;
  const int G = pick_groups(tiles);
  const int grid = (int)((tiles + G - 1) / G);
  const uint8_t* img = static_cast<const uint8_t*>(wp_packed);
  const RowIO io = {nullptr, 0,       1, nullptr, 0, 0, nullptr, 0,
                    nullptr, nullptr, 0, 0, nullptr, nullptr, 0, 0};
  if (M.model == 1) {
    switch (G) {
      case 4: return launch_engine<4, kRollout, 1>(grid, M, B, img, tr, T, t_g0, io, st, s);
      case 2: return launch_engine<2, kRollout, 1>(grid, M, B, img, tr, T, t_g0, io, st, s);
      default: return launch_engine<1, kRollout, 1>(grid, M, B, img, tr, T, t_g0, io, st, s);
    }
  }
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
  const RowIO io = {obs, rows, n, value, M.model == 1 ? 12 : kObs, 1,
                    nullptr, 0, nullptr, nullptr, 0, 0, nullptr, nullptr, 0, 0};
  return launch_rows<kValueRows>(M, static_cast<const uint8_t*>(wv_packed), io, st, s);
}

static bool al32(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 31u) == 0; }

cudaError_t launch_learn_forward_bf16(bool policy, const void* packed, int in_dim, int out_dim,
                                      const uint16_t* x, int ldx, size_t rows, uint16_t* h1,
                                      uint16_t* h2, int ldh, float* out, int ldo, Status* st,
                                      cudaStream_t s) {
  const Model M{};
  RowIO io = {nullptr, rows, 1,   out,     in_dim,  policy ? out_dim : 1, x, ldx, h1, h2,
              ldh,     ldo,  nullptr, nullptr, 0, 0};
  io.wide = ldh % 16 == 0 && al32(h1) && al32(h2) &&
            (!policy || out_dim != kHeadOut || (ldo % 8 == 0 && al32(out)));
  const uint8_t* img = static_cast<const uint8_t*>(packed);
  return policy ? launch_rows<kLearnPolicy>(M, img, io, st, s)
                : launch_rows<kLearnValue>(M, img, io, st, s);
}

cudaError_t launch_learn_backward_bf16(const void* packed, int out_dim, const uint16_t* gy, int ldy,
                                       size_t rows, const uint16_t* h2, const uint16_t* h1, int ldh,
                                       uint16_t* gz2, int ldz2, uint16_t* gz1, int ldz1, Status* st,
                                       cudaStream_t s) {
  const Model M{};
  RowIO io = {nullptr, rows, 1,  nullptr, out_dim, 1,  gy, ldy, gz2, gz1,
              ldz2,    0,    h2, h1,      ldh,     ldz1};
  io.wide = ldz2 % 16 == 0 && ldz1 % 16 == 0 && ldh % 16 == 0 && al32(gz2) && al32(gz1) &&
            al32(h2) && al32(h1);
  return launch_rows<kBackRows>(M, static_cast<const uint8_t*>(packed), io, st, s);
}

cudaError_t launch_forward_bf16(const Model& M, const void* wp_packed, const void* wv_packed,
                                const float* wv_f32, const float* obs, int n, float* head,
                                float* value, Status* st, cudaStream_t s) {
  (void)wv_f32;
  const int od = M.model == 1 ? 12 : kObs;
  const RowIO io = {obs, (size_t)n, 1, head, od, M.policy_out, nullptr, 0,
                    nullptr, nullptr, 0, 0, nullptr, nullptr, 0, 0};
  cudaError_t e = launch_rows<kPolicyRows>(M, static_cast<const uint8_t*>(wp_packed), io, st, s);
  if (e != cudaSuccess || !value) return e;
  const RowIO iov = {obs, (size_t)n, 1, value, od, 1, nullptr, 0,
                     nullptr, nullptr, 0, 0, nullptr, nullptr, 0, 0};
  return launch_rows<kValueRows>(M, static_cast<const uint8_t*>(wv_packed), iov, st, s);
}

}  // namespace auv
