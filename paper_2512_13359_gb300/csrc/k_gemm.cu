// k_gemm.cu -- the learners' dense products (PPO update and SHAC window,
// paper §III-A) on the library's own kernels.
//
//   C[M][N] = beta * C + sum_k A(m, k) B(n, k)
//
// Tensor cores (bf16 or tf32 operands): one CTA computes a 128 x BN tile of
// C over a range of K.  A producer thread streams 128-byte-swizzled tiles of
// A (128 x BK) and B (BN x BK) into a four-stage shared-memory ring with TMA
// (cp.async.bulk.tensor), one thread issues tcgen05.mma into an fp32
// accumulator in tensor memory, and four warps read the accumulator back
// (tcgen05.ld) and write C, or an fp32 partial when K is split over CTAs.
// BK is 128 bytes of K per row: 64 bf16 or 32 tf32 elements.
//
// Operand tiles in shared memory are the canonical 128-byte-swizzle
// layouts of the tensor-core descriptors:
//  - K-major (row r of the tile, K contiguous): one TMA box of BK x rows;
//    row r at r * 128 bytes, 8-row groups 1024 bytes apart (SBO); an MMA's
//    K-step advances the start address by 32 bytes.
//  - MN-major (K row kk, the M or N index contiguous): boxes of 128 bytes of
//    M/N x BK rows, one per 128 bytes of M/N, BK * 128 bytes apart (LBO);
//    8 K rows form a 1024-byte group (SBO); an MMA's K-step (32 bytes of
//    K) advances the start address by 4096 / element-size bytes.
//
// fp32 operands without tensor cores (the exact mode): a register-blocked CUDA-core
// kernel with the same operand layouts and the same split-K.
//
// Split-K: partial tiles go to ws[z][M_pad][N_pad] (fp32); k_reduce adds
// them in a fixed order (eight interleaved partial sums over z, then those
// eight in order) and applies beta and the output type.
#include <cuda.h>

#include <algorithm>
#include <mutex>

#include "auv_device.cuh"
#include "auv_gemm.h"
#include "auvenv.h"
#include "tc_ptx.cuh"

namespace auv {
namespace gemm {
namespace {

constexpr int kMaxStages = 4;
constexpr int kBM = 128;
constexpr uint64_t kWaitLimitNs = 2000000000ull;

// ---------------------------------------------------------------------------
// device helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes "
      "[%0], [%1, {%2, %3}], [%4];" ::"r"(tc::smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(tc::smem_u32(bar))
      : "memory");
}

// Shared-memory descriptor with both byte offsets (128-byte swizzle).
__device__ __forceinline__ uint64_t desc_sw128(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1u << 46;                       // descriptor version
  d |= (uint64_t)2u << 61;                       // 128-byte swizzle
  return d;
}

// Instruction descriptor: D fp32, A/B bf16 (kind::f16) or tf32 (kind::tf32),
// major-ness of A (bit 15) and B (bit 16): 1 = MN-major.
__host__ __device__ constexpr uint32_t idesc(bool tf32, bool a_mn, bool b_mn, int M, int N) {
  return (1u << 4) | ((tf32 ? 2u : 1u) << 7) | ((tf32 ? 2u : 1u) << 10) |
         ((a_mn ? 1u : 0u) << 15) | ((b_mn ? 1u : 0u) << 16) | ((uint32_t)(N >> 3) << 17) |
         ((uint32_t)(M >> 4) << 24);
}

template <bool TF32>
__device__ __forceinline__ void mma(uint32_t d, uint64_t a, uint64_t b, uint32_t id, uint32_t acc) {
  if constexpr (TF32) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}" ::"r"(d),
        "l"(a), "l"(b), "r"(id), "r"(acc)
        : "memory");
  } else {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d),
        "l"(a), "l"(b), "r"(id), "r"(acc)
        : "memory");
  }
}

struct TcArgs {
  int M, N, K;
  int chunks_per_split;   // K chunks of BK per CTA along z
  void* C;
  int ldc;
  int c_bf16;
  float beta;
  float* ws;              // split partials, or null (write C directly)
  int n_pad, m_pad;
  Status* st;
  int vec;                // C base and ldc allow 16-byte (1) or 32-byte (2) row segments
  int ws_wide;            // ws 32-byte aligned: partial rows as whole 32-byte sectors
};

// 8 floats to a 32-byte aligned address with one 256-bit store (a whole L2
// sector; a thread writing its own row otherwise fills half a sector per
// access).
__device__ __forceinline__ void st_f32x8(float* p, const uint32_t* v) {
  asm volatile("st.global.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(p), "r"(v[0]),
               "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7])
               : "memory");
}

// BN = 320 (for N in (256, 320]: the weight gradients' 264 augmented
// columns) is one N = 256 and one N = 64 MMA per K-step, in a three-stage
// ring; the other widths are one MMA in a four-stage ring.
template <bool TF32, bool A_MN, bool B_MN, int BN>
struct Tile {
  static constexpr int kEs = TF32 ? 4 : 2;
  static constexpr int kBK = 128 / kEs;                 // K elements per stage
  static constexpr int kStages = BN > 256 ? 3 : 4;
  static constexpr uint32_t kABytes = kBM * 128;        // 128 rows (or BK K-rows x 128 B x 128/E)
  static constexpr uint32_t kBBytes = BN * 128;
  static constexpr uint32_t kStage = kABytes + kBBytes;
  static constexpr uint32_t kSmem = kStages * kStage + 256 + 1024;
  static constexpr int kElemsPer128 = 128 / kEs;        // M/N elements per MN-major box
  static constexpr int kBoxRows = BN > 256 ? 64 : BN;   // K-major B: rows per TMA box
  static constexpr uint32_t kTmemCols = BN > 256 ? 512 : BN;
};

struct Bars {
  uint64_t full[kMaxStages];
  uint64_t empty[kMaxStages];
  uint64_t acc_full;
  uint32_t tmem_base;
  int abort;
};

// One CTA: warps 0-3 epilogue (tensor-memory lanes 0..127 = rows), warp 4
// TMA producer, warp 5 MMA issuer and tensor-memory owner.
template <bool TF32, bool A_MN, bool B_MN, int BN>
__global__ void __launch_bounds__(192, 1)
k_gemm_tc(const __grid_constant__ CUtensorMap map_a, const __grid_constant__ CUtensorMap map_b,
          TcArgs args) {
  using TL = Tile<TF32, A_MN, B_MN, BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023u) & ~(uintptr_t)1023u);
  constexpr int kStages = TL::kStages;
  Bars* bar = reinterpret_cast<Bars*>(smem + kStages * TL::kStage);
  volatile int* abort = &bar->abort;
  const int tid = threadIdx.x, warp = tid >> 5;
  const int m0 = blockIdx.x * kBM, n0 = blockIdx.y * BN;
  const int n_chunks_total = (args.K + TL::kBK - 1) / TL::kBK;
  const int c0 = blockIdx.z * args.chunks_per_split;
  const int c1 = min(n_chunks_total, c0 + args.chunks_per_split);
  const int n_chunks = max(0, c1 - c0);

  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      tc::mbar_init(&bar->full[s], 1);
      tc::mbar_init(&bar->empty[s], 1);
    }
    tc::mbar_init(&bar->acc_full, 1);
    bar->abort = 0;
    tc::mbar_fence_init();
  }
  if (warp == 5) {
    tc::tmem_alloc(&bar->tmem_base, TL::kTmemCols);
    tc::tmem_relinquish();
  }
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = bar->tmem_base;
  const uint32_t s_base = tc::smem_u32(smem);

  if (warp == 4) {
    // ---- producer: TMA tiles of A and B into the ring ----
    if ((tid & 31) == 0) {
      for (int c = 0; c < n_chunks; ++c) {
        const int s = c % kStages;
        if (c >= kStages &&
            !tc::mbar_wait(&bar->empty[s], (uint32_t)((c / kStages) - 1) & 1u, abort, kWaitLimitNs))
          break;
        uint8_t* a_dst = smem + s * TL::kStage;
        uint8_t* b_dst = a_dst + TL::kABytes;
        tc::mbar_arrive_expect_tx(&bar->full[s], TL::kStage);
        const int k = (c0 + c) * TL::kBK;
        if (A_MN) {
#pragma unroll
          for (int j = 0; j < kBM / TL::kElemsPer128; ++j)
            tma_load_2d(a_dst + j * (TL::kBK * 128), &map_a, m0 + j * TL::kElemsPer128, k, &bar->full[s]);
        } else {
          tma_load_2d(a_dst, &map_a, k, m0, &bar->full[s]);
        }
        if (B_MN) {
#pragma unroll
          for (int j = 0; j < BN / TL::kElemsPer128; ++j)
            tma_load_2d(b_dst + j * (TL::kBK * 128), &map_b, n0 + j * TL::kElemsPer128, k, &bar->full[s]);
        } else {
#pragma unroll
          for (int j = 0; j < BN / TL::kBoxRows; ++j)
            tma_load_2d(b_dst + j * (TL::kBoxRows * 128), &map_b, k, n0 + j * TL::kBoxRows,
                        &bar->full[s]);
        }
      }
    }
    __syncwarp();
  } else if (warp == 5) {
    // ---- MMA issue ----
    if ((tid & 31) == 0) {
      constexpr uint32_t kId = idesc(TF32, A_MN, B_MN, kBM, BN > 256 ? 256 : BN);
      constexpr uint32_t kId2 = idesc(TF32, A_MN, B_MN, kBM, BN > 256 ? BN - 256 : 16);
      // second MMA of a 320-wide tile: B from column 256 (MN-major: the fifth
      // 128-byte block of bf16; K-major: row 256)
      constexpr uint32_t kB2 = B_MN ? (256 / TL::kElemsPer128) * (TL::kBK * 128) : 256 * 128;
      constexpr uint32_t kLbo = TL::kBK * 128;          // MN-major: between 128-byte M/N blocks
      constexpr uint32_t kKStepMn = 4096 / TL::kEs;     // MN-major: bytes per 32 bytes of K
      bool ok = true;
      for (int c = 0; c < n_chunks && ok; ++c) {
        const int s = c % kStages;
        ok = tc::mbar_wait(&bar->full[s], (uint32_t)(c / kStages) & 1u, abort, kWaitLimitNs);
        if (!ok) break;
        tc::tc_fence_after();
        const uint32_t a0 = s_base + s * TL::kStage, b0 = a0 + TL::kABytes;
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
          const uint64_t da = A_MN ? desc_sw128(a0 + kk * kKStepMn, kLbo, 1024)
                                   : desc_sw128(a0 + kk * 32, 16, 1024);
          const uint64_t db = B_MN ? desc_sw128(b0 + kk * kKStepMn, kLbo, 1024)
                                   : desc_sw128(b0 + kk * 32, 16, 1024);
          mma<TF32>(tmem, da, db, kId, (c > 0 || kk > 0) ? 1u : 0u);
          if constexpr (BN > 256) {
            const uint64_t db2 = B_MN ? desc_sw128(b0 + kB2 + kk * kKStepMn, kLbo, 1024)
                                      : desc_sw128(b0 + kB2 + kk * 32, 16, 1024);
            mma<TF32>(tmem + 256, da, db2, kId2, (c > 0 || kk > 0) ? 1u : 0u);
          }
        }
        tc::mma_commit(&bar->empty[s]);
      }
      tc::mma_commit(&bar->acc_full);
    }
    __syncwarp();
  } else {
    // ---- epilogue: row m0 + tid of the tile, BN columns in chunks of 32 ----
    const bool ok = n_chunks > 0 && tc::mbar_wait(&bar->acc_full, 0, abort, kWaitLimitNs);
    tc::tc_fence_after();
    const int row = m0 + tid;
    const uint32_t lane_addr = tmem + ((uint32_t)(warp * 32) << 16);
#pragma unroll 1
    for (int j = 0; j < BN / 32; ++j) {
      uint32_t acc[32];
      tc::tmem_ld32(lane_addr + j * 32, acc);
      tc::tmem_ld_wait(acc);
      if (!ok) {
#pragma unroll
        for (int q = 0; q < 32; ++q) acc[q] = 0u;   // no K in range (or a timed-out wait)
      }
      const int nb = n0 + j * 32;
      if (args.ws) {
        // partials of the rows and 32-column groups the reduction reads
        if (row < args.M && nb < args.N) {
          float* dst = args.ws + ((size_t)blockIdx.z * args.m_pad + row) * args.n_pad + nb;
          if (args.ws_wide) {
#pragma unroll
            for (int q = 0; q < 4; ++q) st_f32x8(dst + 8 * q, acc + 8 * q);
          } else {
            float4* d4 = reinterpret_cast<float4*>(dst);
#pragma unroll
            for (int q = 0; q < 8; ++q)
              d4[q] = make_float4(__uint_as_float(acc[4 * q]), __uint_as_float(acc[4 * q + 1]),
                                  __uint_as_float(acc[4 * q + 2]), __uint_as_float(acc[4 * q + 3]));
          }
        }
      } else if (row < args.M && args.beta == 0.0f && nb + 32 <= args.N && args.vec) {
        // whole 32-column segment, 16-byte aligned rows: vector stores
        // (32-byte aligned rows: whole sectors)
        if (args.c_bf16) {
          uint16_t* crow = static_cast<uint16_t*>(args.C) + (size_t)row * args.ldc + nb;
          uint32_t w[16];
#pragma unroll
          for (int e = 0; e < 16; ++e)
            w[e] = tc::pack_bf16x2(__uint_as_float(acc[2 * e]), __uint_as_float(acc[2 * e + 1]));
          if (args.vec == 2) {
            st_f32x8(reinterpret_cast<float*>(crow), w);
            st_f32x8(reinterpret_cast<float*>(crow + 16), w + 8);
          } else {
            uint4* dst = reinterpret_cast<uint4*>(crow);
#pragma unroll
            for (int q = 0; q < 4; ++q) dst[q] = make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
          }
        } else if (args.vec == 2) {
          float* crow = static_cast<float*>(args.C) + (size_t)row * args.ldc + nb;
#pragma unroll
          for (int q = 0; q < 4; ++q) st_f32x8(crow + 8 * q, acc + 8 * q);
        } else {
          float4* dst = reinterpret_cast<float4*>(static_cast<float*>(args.C) +
                                                  (size_t)row * args.ldc + nb);
#pragma unroll
          for (int q = 0; q < 8; ++q)
            dst[q] = make_float4(__uint_as_float(acc[4 * q]), __uint_as_float(acc[4 * q + 1]),
                                 __uint_as_float(acc[4 * q + 2]), __uint_as_float(acc[4 * q + 3]));
        }
      } else if (row < args.M) {
        if (args.c_bf16) {
          uint16_t* crow = static_cast<uint16_t*>(args.C) + (size_t)row * args.ldc;
#pragma unroll
          for (int q = 0; q < 32; ++q) {
            const int n = nb + q;
            if (n < args.N) {
              float v = __uint_as_float(acc[q]);
              if (args.beta != 0.0f)
                v = fmaf(args.beta, __uint_as_float((uint32_t)crow[n] << 16), v);
              crow[n] = (uint16_t)(tc::pack_bf16x2(v, 0.0f) & 0xFFFFu);
            }
          }
        } else {
          float* crow = static_cast<float*>(args.C) + (size_t)row * args.ldc;
#pragma unroll
          for (int q = 0; q < 32; ++q) {
            const int n = nb + q;
            if (n < args.N) {
              float v = __uint_as_float(acc[q]);
              if (args.beta != 0.0f) v = fmaf(args.beta, crow[n], v);
              crow[n] = v;
            }
          }
        }
      }
    }
  }
  tc::tc_fence_before();
  __syncthreads();
  if (tid == 0 && bar->abort) {
    atomicAdd(&args.st->timeouts, 1);
    atomicCAS(&args.st->code, 0, -4);
  }
  if (warp == 5) {
    tc::tc_fence_after();
    tc::tmem_dealloc(tmem, TL::kTmemCols);
  }
}

// fp32 CUDA-core GEMM: a BM x 128 tile of C per CTA (BM = 128, or 32 for
// the few-row weight gradients of the output layers), 256 threads as 16 x 16
// with BM/16 x 8 outputs each (BM = 128: rows ty*4 .. +3 and 64 + ty*4 .. +3,
// columns likewise, so shared-memory reads are float4; BM = 32: rows ty*2,
// ty*2 + 1), K in slices of 8 through double-buffered shared memory that
// holds both operands M/N-fastest (As[k][m], Bs[k][n]) whichever way they
// are stored.  Rows are padded by 4 floats: the K-major loads' stores (8 k of
// 4 rows per warp) then land in 32 distinct banks, and row starts stay
// 16-byte aligned.
template <int BM, bool A_MN, bool B_MN>
__global__ void __launch_bounds__(256, 2)
k_gemm_fp32(int M, int N, int K, const float* __restrict__ A, int lda, const float* __restrict__ B,
            int ldb, int chunks_per_split, void* C, int ldc, float beta, float* ws, int m_pad,
            int n_pad) {
  constexpr int RM = BM / 16, QA = BM / 32;
  __shared__ __align__(16) float As[2][8][BM + 4];
  __shared__ __align__(16) float Bs[2][8][132];
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int m0 = blockIdx.x * BM, n0 = blockIdx.y * 128;
  const int k_begin = blockIdx.z * chunks_per_split * 8;
  const int k_end = min(K, k_begin + chunks_per_split * 8);
  // element e of a ROWS x 8 slice: (row, k) with consecutive threads along
  // the stored-contiguous index
  auto coord = [](int e, int rows, bool mn, int& r, int& kk) {
    if (mn) { kk = e / rows; r = e % rows; } else { r = e >> 3; kk = e & 7; }
  };
  auto load = [&](const float* X, int ld, bool mn, int rows, int r0, int R, int kb, float* v, int q_n) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      if (q >= q_n) break;
      int r, kk;
      coord(tid + 256 * q, rows, mn, r, kk);
      const int rr = r0 + r, k = kb + kk;
      v[q] = (rr < R && k < k_end) ? (mn ? X[(size_t)k * ld + rr] : X[(size_t)rr * ld + k]) : 0.0f;
    }
  };
  auto store = [&](float* S, int stride, bool mn, int rows, const float* v, int q_n) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      if (q >= q_n) break;
      int r, kk;
      coord(tid + 256 * q, rows, mn, r, kk);
      S[kk * stride + r] = v[q];
    }
  };
  float acc[RM][8] = {};
  float va[4], vb[4];
  int buf = 0;
  if (k_begin < k_end) {
    load(A, lda, A_MN, BM, m0, M, k_begin, va, QA);
    load(B, ldb, B_MN, 128, n0, N, k_begin, vb, 4);
    store(&As[0][0][0], BM + 4, A_MN, BM, va, QA);
    store(&Bs[0][0][0], 132, B_MN, 128, vb, 4);
  }
  __syncthreads();
  for (int kb = k_begin; kb < k_end; kb += 8) {
    const bool more = kb + 8 < k_end;
    if (more) {                                   // next slice in flight during this one
      load(A, lda, A_MN, BM, m0, M, kb + 8, va, QA);
      load(B, ldb, B_MN, 128, n0, N, kb + 8, vb, 4);
    }
#pragma unroll
    for (int kk = 0; kk < 8; ++kk) {
      float a[RM];
      if constexpr (BM == 128) {
        const float4 a0 = *reinterpret_cast<const float4*>(&As[buf][kk][ty * 4]);
        const float4 a1 = *reinterpret_cast<const float4*>(&As[buf][kk][64 + ty * 4]);
        a[0] = a0.x; a[1] = a0.y; a[2] = a0.z; a[3] = a0.w;
        a[4] = a1.x; a[5] = a1.y; a[6] = a1.z; a[7] = a1.w;
      } else {
        const float2 a0 = *reinterpret_cast<const float2*>(&As[buf][kk][ty * 2]);
        a[0] = a0.x; a[1] = a0.y;
      }
      const float4 b0 = *reinterpret_cast<const float4*>(&Bs[buf][kk][tx * 4]);
      const float4 b1 = *reinterpret_cast<const float4*>(&Bs[buf][kk][64 + tx * 4]);
      const float b[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
      for (int i = 0; i < RM; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    if (more) {
      store(&As[buf ^ 1][0][0], BM + 4, A_MN, BM, va, QA);
      store(&Bs[buf ^ 1][0][0], 132, B_MN, 128, vb, 4);
    }
    __syncthreads();
    buf ^= 1;
  }
#pragma unroll
  for (int i = 0; i < RM; ++i) {
    const int m = m0 + (BM == 128 ? (i < 4 ? ty * 4 + i : 64 + ty * 4 + i - 4) : ty * 2 + i);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int n = n0 + (j < 4 ? tx * 4 + j : 64 + tx * 4 + j - 4);
      if (ws) {   // partials of the elements the reduction reads
        if (m < M && n < N) ws[((size_t)blockIdx.z * m_pad + m) * n_pad + n] = acc[i][j];
      } else if (m < M && n < N) {
        float* c = static_cast<float*>(C) + (size_t)m * ldc + n;
        *c = beta != 0.0f ? fmaf(beta, *c, acc[i][j]) : acc[i][j];
      }
    }
  }
}

// C = beta C + sum_z ws[z], fp32 or bf16 output.  A weight gradient has a
// few tens of thousands of elements and tens of splits, so one thread per
// element summing every split in turn left the kernel bound by load latency
// at under two blocks per SM.  Here a block of 256 threads covers 128
// consecutive elements (32 groups of four, 16-byte loads) for 8 groups of
// splits: thread (g, l) adds the partials z = g, g + 8, g + 16, ... of its
// four elements in increasing z, and the eight group sums are then added in
// the order g = 0..7: a fixed order, the same on every run.
constexpr int kRedGroups = 8;
constexpr int kRedQuads = 32;
__global__ void __launch_bounds__(kRedGroups * kRedQuads)
k_reduce(int M, int N, int splits, const float* __restrict__ ws, int m_pad, int n_pad, void* C,
         int ldc, int c_bf16, float beta) {
  __shared__ float4 part[kRedGroups][kRedQuads];
  const int lane = threadIdx.x % kRedQuads, grp = threadIdx.x / kRedQuads;
  const int qpr = (N + 3) / 4;   // groups of four per row (n_pad is a multiple of 128)
  const long quad = (long)blockIdx.x * kRedQuads + lane;
  const bool live = quad < (long)M * qpr;
  const int m = live ? (int)(quad / qpr) : 0, n = live ? (int)(quad % qpr) * 4 : 0;
  const size_t zs = (size_t)m_pad * n_pad;
  const float* src = ws + (size_t)m * n_pad + n;
  // 16-byte loads when the workspace is 16-byte aligned (every offset here
  // is a multiple of four floats), four scalar loads otherwise
  const bool vec = (reinterpret_cast<uintptr_t>(ws) & 15u) == 0;
  auto load4 = [&](const float* a) {
    return vec ? __ldcs(reinterpret_cast<const float4*>(a))
               : make_float4(__ldcs(a), __ldcs(a + 1), __ldcs(a + 2), __ldcs(a + 3));
  };
  float4 v = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
  if (live) {
    constexpr int kU = 4;   // loads in flight per thread
    for (int z0 = grp; z0 < splits; z0 += kRedGroups * kU) {
      float4 p[kU];
#pragma unroll
      for (int q = 0; q < kU; ++q) {
        const int z = z0 + q * kRedGroups;
        p[q] = z < splits ? load4(src + (size_t)z * zs) : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
      }
#pragma unroll
      for (int q = 0; q < kU; ++q)
        if (z0 + q * kRedGroups < splits) {
          v.x += p[q].x;
          v.y += p[q].y;
          v.z += p[q].z;
          v.w += p[q].w;
        }
    }
  }
  part[grp][lane] = v;
  __syncthreads();
  if (grp != 0 || !live) return;
  float4 s = part[0][lane];
#pragma unroll
  for (int g = 1; g < kRedGroups; ++g) {
    const float4 u = part[g][lane];
    s.x += u.x;
    s.y += u.y;
    s.z += u.z;
    s.w += u.w;
  }
  const float r[4] = {s.x, s.y, s.z, s.w};
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    if (n + j >= N) break;
    float x = r[j];
    if (c_bf16) {
      uint16_t* c = static_cast<uint16_t*>(C) + (size_t)m * ldc + n + j;
      if (beta != 0.0f) x = fmaf(beta, __uint_as_float((uint32_t)*c << 16), x);
      *c = (uint16_t)(tc::pack_bf16x2(x, 0.0f) & 0xFFFFu);
    } else {
      float* c = static_cast<float*>(C) + (size_t)m * ldc + n + j;
      *c = beta != 0.0f ? fmaf(beta, *c, x) : x;
    }
  }
}

// An MN-major fp32 operand (element (r, k) at k * ld + r) copied K-major:
// out[r * ldo + k], 32 x 32 tiles through shared memory, both sides coalesced.
// (The tf32 tensor-core path reads its operands K-major.)
__global__ void k_transpose(int R, int K, const float* __restrict__ in, int ld, float* out,
                            int ldo) {
  __shared__ float tile[32][33];
  const int r0 = blockIdx.x * 32, k0 = blockIdx.y * 32;
  for (int j = threadIdx.y; j < 32; j += 8) {
    const int k = k0 + j, r = r0 + threadIdx.x;
    tile[j][threadIdx.x] = (k < K && r < R) ? in[(size_t)k * ld + r] : 0.0f;
  }
  __syncthreads();
  for (int j = threadIdx.y; j < 32; j += 8) {
    const int r = r0 + j, k = k0 + threadIdx.x;
    if (r < R && k < ldo) out[(size_t)r * ldo + k] = k < K ? tile[threadIdx.x][j] : 0.0f;
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
using EncodeFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                              const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                              const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                              CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeFn encode_fn() {
  static EncodeFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeFn>(p);
    else
      cudaGetLastError();
  });
  return fn;
}

// 2-D map of a stored operand: inner dimension (contiguous) and outer
// dimension, rows ld elements apart; a box of 128 bytes x box_outer rows.
bool make_map(CUtensorMap* map, bool tf32, const void* ptr, uint64_t inner, uint64_t outer, int ld,
              uint32_t box_outer) {
  EncodeFn fn = encode_fn();
  if (!fn) return false;
  const int es = tf32 ? 4 : 2;
  const cuuint64_t dims[2] = {inner, outer};
  const cuuint64_t strides[1] = {(cuuint64_t)ld * es};
  const cuuint32_t box[2] = {(cuuint32_t)(128 / es), box_outer};
  const cuuint32_t estr[2] = {1, 1};
  // tf32: the copy rounds each fp32 element to tf32 (nearest), as a tf32
  // GEMM rounds its operands, instead of the MMA dropping the low bits
  return fn(map, tf32 ? CU_TENSOR_MAP_DATA_TYPE_TFLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
            const_cast<void*>(ptr), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int sm_count_dev() {
  int dev = 0, v = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v <= 0) {
    cudaGetLastError();
    return 148;
  }
  return v;
}

struct Plan {
  int bm, bn, bk;        // tile and K-chunk sizes
  int tiles_m, tiles_n;
  int chunks, per_split, splits;
  int m_pad, n_pad;
};

Plan plan(Prec prec, int M, int N, int K) {
  Plan p;
  if (prec == kFp32) {
    p.bm = M <= 32 ? 32 : 128;
    p.bn = 128;
    p.bk = 8;
  } else {
    p.bm = kBM;
    // 320-wide tiles (one CTA over the weight gradients' 264 augmented
    // columns: the other operand read once instead of three times) pay when
    // there are at least two M-tiles; with one, three 128-wide tiles keep more
    // CTAs per K-range (measured 28.1 against 37.9 us for 256 x 264 x 65,536,
    // 25.4 against 21.4 us for 16 x 264 x 65,536)
    p.bn = (N > 128 && N <= 256) ? 256 : ((N > 256 && N <= 320 && M > kBM) ? 320 : 128);
    p.bk = prec == kTf32 ? 32 : 64;
  }
  p.tiles_m = (M + p.bm - 1) / p.bm;
  p.tiles_n = (N + p.bn - 1) / p.bn;
  p.chunks = std::max(1, (K + p.bk - 1) / p.bk);
  const int tiles = p.tiles_m * p.tiles_n;
  // CTAs wanted: one per SM for the tensor-core kernel, two for the
  // CUDA-core one (two 256-thread CTAs resident per SM hide its loads)
  const int sms = sm_count_dev() * (prec == kFp32 ? 2 : 1);
  int want = tiles >= sms / 2 ? 1 : (sms + tiles - 1) / tiles;
  // at least 4 K-chunks per CTA, at most one split per chunk
  want = std::max(1, std::min(want, p.chunks / 4));
  p.per_split = (p.chunks + want - 1) / want;
  p.splits = (p.chunks + p.per_split - 1) / p.per_split;
  p.m_pad = p.tiles_m * p.bm;
  p.n_pad = p.tiles_n * p.bn;
  return p;
}

template <bool TF32, bool A_MN, bool B_MN, int BN>
cudaError_t launch_tc(const Plan& P, const CUtensorMap& ma, const CUtensorMap& mb,
                      const TcArgs& a, cudaStream_t s) {
  using TL = Tile<TF32, A_MN, B_MN, BN>;
  auto kern = k_gemm_tc<TF32, A_MN, B_MN, BN>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, TL::kSmem);
  if (e != cudaSuccess) return e;
  kern<<<dim3(P.tiles_m, P.tiles_n, P.splits), 192, TL::kSmem, s>>>(ma, mb, a);
  return cudaGetLastError();
}

template <bool TF32, int BN>
cudaError_t dispatch_major(bool a_mn, bool b_mn, const Plan& P, const CUtensorMap& ma,
                           const CUtensorMap& mb, const TcArgs& a, cudaStream_t s) {
  if (a_mn && b_mn) return launch_tc<TF32, true, true, BN>(P, ma, mb, a, s);
  if (a_mn) return launch_tc<TF32, true, false, BN>(P, ma, mb, a, s);
  if (b_mn) return launch_tc<TF32, false, true, BN>(P, ma, mb, a, s);
  return launch_tc<TF32, false, false, BN>(P, ma, mb, a, s);
}

bool tma_ok(const Operand& o, int es) {
  return (reinterpret_cast<uintptr_t>(o.ptr) & 15u) == 0 && ((size_t)o.ld * es) % 16 == 0;
}

}  // namespace

// tf32 with MN-major operands: K-major copies of A and B ahead of the partials.
size_t transposed_floats(int rows, int K) {
  return ((size_t)rows * ((K + 3) & ~3) + 63) & ~(size_t)63;   // 256-byte multiples
}

size_t workspace_bytes(int M, int N, int K) {
  size_t best = 0;
  for (Prec p : {kFp32, kTf32, kBf16}) {
    const Plan P = plan(p, M, N, K);
    size_t b = P.splits > 1 ? (size_t)P.splits * P.m_pad * P.n_pad * sizeof(float) : 0;
    if (p == kTf32) b += (transposed_floats(M, K) + transposed_floats(N, K)) * sizeof(float);
    best = std::max(best, b);
  }
  return best;
}

cudaError_t launch(Prec prec, int M, int N, int K, const Operand& A_in, const Operand& B_in,
                   void* C, int ldc, bool c_bf16, float beta, float* ws, size_t ws_bytes,
                   Status* st, cudaStream_t s) {
  if (M <= 0 || N <= 0) return cudaSuccess;
  Operand A = A_in, B = B_in;
  if (prec == kTf32 && (A.mn_major || B.mn_major)) {
    // kind::tf32 reads K-major operands: transpose the MN-major ones into
    // the front of the workspace, 256-byte aligned
    const size_t need = (transposed_floats(M, K) + transposed_floats(N, K)) * sizeof(float);
    if (!ws || ws_bytes < need) return cudaErrorInvalidValue;
    float* dst = ws;
    for (Operand* o : {&A, &B}) {
      const int rows = o == &A ? M : N;
      if (o->mn_major) {
        const int ldo = (K + 3) & ~3;
        k_transpose<<<dim3((rows + 31) / 32, (ldo + 31) / 32), dim3(32, 8), 0, s>>>(
            rows, K, static_cast<const float*>(o->ptr), o->ld, dst, ldo);
        const cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
        *o = {dst, ldo, false};
      }
      dst += transposed_floats(rows, K);
    }
    const size_t used = (size_t)(dst - ws) * sizeof(float);
    ws = dst;
    ws_bytes -= used;
  }
  Plan P = plan(prec, M, N, K);
  const size_t need = (size_t)P.splits * P.m_pad * P.n_pad * sizeof(float);
  if (P.splits > 1 && (!ws || ws_bytes < need)) {
    // no room for partials: one CTA per tile over the whole K
    P.per_split = std::max(1, P.chunks);
    P.splits = 1;
  }
  float* part = P.splits > 1 ? ws : nullptr;
  cudaError_t e = cudaSuccess;
  if (prec == kFp32) {
    const dim3 grid(P.tiles_m, P.tiles_n, P.splits);
    const float* a = static_cast<const float*>(A.ptr);
    const float* b = static_cast<const float*>(B.ptr);
#define AUV_FP32_GEMM(TM, AM, BM)                                                           \
  k_gemm_fp32<TM, AM, BM><<<grid, 256, 0, s>>>(M, N, K, a, A.ld, b, B.ld, P.per_split, C, ldc, \
                                               beta, part, P.m_pad, P.n_pad)
#define AUV_FP32_MAJOR(TM)                                         \
  if (A.mn_major && B.mn_major) AUV_FP32_GEMM(TM, true, true);     \
  else if (A.mn_major) AUV_FP32_GEMM(TM, true, false);             \
  else if (B.mn_major) AUV_FP32_GEMM(TM, false, true);             \
  else AUV_FP32_GEMM(TM, false, false)
    if (P.bm == 32) { AUV_FP32_MAJOR(32); }
    else { AUV_FP32_MAJOR(128); }
#undef AUV_FP32_MAJOR
#undef AUV_FP32_GEMM
    e = cudaGetLastError();
  } else {
    const bool tf32 = prec == kTf32;
    const int es = tf32 ? 4 : 2;
    if (!tma_ok(A, es) || !tma_ok(B, es)) return cudaErrorInvalidValue;
    const int bk = P.bk;
    CUtensorMap ma, mb;
    // K-major: inner = K, outer = rows (box: 128 B of K x tile rows);
    // MN-major: inner = rows, outer = K (box: 128 B of rows x BK).
    const bool ok_a = A.mn_major ? make_map(&ma, tf32, A.ptr, M, K, A.ld, bk)
                                 : make_map(&ma, tf32, A.ptr, K, M, A.ld, kBM);
    const bool ok_b = B.mn_major ? make_map(&mb, tf32, B.ptr, N, K, B.ld, bk)
                                 : make_map(&mb, tf32, B.ptr, K, N, B.ld, P.bn > 256 ? 64 : P.bn);
    if (!ok_a || !ok_b) return cudaErrorInvalidValue;
    const int ces = c_bf16 ? 2 : 4;
    const int vec = (reinterpret_cast<uintptr_t>(C) % 32 == 0 && ((size_t)ldc * ces) % 32 == 0)
                        ? 2
                        : ((reinterpret_cast<uintptr_t>(C) % 16 == 0 && ((size_t)ldc * ces) % 16 == 0) ? 1 : 0);
    const int ws_wide = reinterpret_cast<uintptr_t>(part) % 32 == 0 ? 1 : 0;
    TcArgs a = {M,     N,      K,       P.per_split, C,  ldc,    c_bf16 ? 1 : 0,
                beta,  part,   P.n_pad, P.m_pad,     st, vec,    ws_wide};
    if (tf32)
      e = P.bn == 320   ? dispatch_major<true, 320>(A.mn_major, B.mn_major, P, ma, mb, a, s)
          : P.bn == 256 ? dispatch_major<true, 256>(A.mn_major, B.mn_major, P, ma, mb, a, s)
                        : dispatch_major<true, 128>(A.mn_major, B.mn_major, P, ma, mb, a, s);
    else
      e = P.bn == 320   ? dispatch_major<false, 320>(A.mn_major, B.mn_major, P, ma, mb, a, s)
          : P.bn == 256 ? dispatch_major<false, 256>(A.mn_major, B.mn_major, P, ma, mb, a, s)
                        : dispatch_major<false, 128>(A.mn_major, B.mn_major, P, ma, mb, a, s);
  }
  if (e != cudaSuccess || !part) return e;
  const size_t quads = (size_t)M * ((N + 3) / 4);
  k_reduce<<<(unsigned)((quads + kRedQuads - 1) / kRedQuads), kRedGroups * kRedQuads, 0, s>>>(
      M, N, P.splits, part, P.m_pad, P.n_pad, C, ldc, c_bf16 ? 1 : 0, beta);
  return cudaGetLastError();
}

}  // namespace gemm
}  // namespace auv

// ---------------------------------------------------------------------------
// C ABI (include/auvenv.h): the learners' dense product on its own
// ---------------------------------------------------------------------------
extern "C" size_t auv_gemm_workspace_bytes(int M, int N, int K) {
  return (M > 0 && N > 0 && K > 0) ? auv::gemm::workspace_bytes(M, N, K) : 0;
}

extern "C" int auv_gemm(uint32_t precision, int M, int N, int K, const void* A, int lda, int a_mn,
                        const void* B, int ldb, int b_mn, void* C, int ldc, int c_bf16, float beta,
                        void* workspace, size_t workspace_bytes, auv_status* status, void* stream) {
  if (precision > AUV_PPO_BF16 || M < 1 || N < 1 || K < 1 || !A || !B || !C || !status)
    return AUV_ERR_INVALID;
  if ((precision == AUV_PPO_FP32 && c_bf16) || lda < 1 || ldb < 1 || ldc < N ||
      lda < (a_mn ? M : K) || ldb < (b_mn ? N : K))
    return AUV_ERR_INVALID;
  static_assert(sizeof(auv::Status) == sizeof(auv_status), "status block layout");
  const auv::gemm::Operand a = {A, lda, a_mn != 0}, b = {B, ldb, b_mn != 0};
  const cudaError_t e = auv::gemm::launch(static_cast<auv::gemm::Prec>(precision), M, N, K, a, b, C,
                                          ldc, c_bf16 != 0, beta, static_cast<float*>(workspace),
                                          workspace ? workspace_bytes : 0,
                                          reinterpret_cast<auv::Status*>(status),
                                          static_cast<cudaStream_t>(stream));
  if (e == cudaErrorInvalidValue) return AUV_ERR_SIZE;
  return e == cudaSuccess ? AUV_OK : AUV_ERR_CUDA;
}
