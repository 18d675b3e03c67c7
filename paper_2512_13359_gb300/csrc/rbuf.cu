// rbuf.cu -- the off-policy pieces: a device replay buffer of transitions for
// DroQ (paper §III-A: off-policy learning from replayed experience; Hiraoka
// et al. 2022) and the inverse thruster allocation used at deployment (paper
// §V-B: body-frame wrench -> thruster commands through the allocation matrix).
//
// Replay buffer: a ring of `capacity` transitions stored sample-major, one
// array per field (obs [C][D], act [C][A], rew [C], next_obs [C][D],
// done [C]), so that a sampled transition is a few contiguous rows.
// Insertion takes a rollout's feature-major trajectory [T][D][N] and
// transposes it through shared memory: each block moves 32 consecutive envs
// of one step, reading 32-wide coalesced rows and writing 32 consecutive
// slots (one contiguous span of 32 x D floats unless the ring wraps).
// Sampling draws indices from a counter-based generator (Philox4x32-10 at
// counter (b, 0x52420000, draw), key = seed; index = floor(word * size /
// 2^32)) and gathers the rows.
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <new>

#include "auv_kernels.h"
#include "auvenv.h"

struct auv_rbuf {
  uint32_t D, A;
  uint64_t C;
  int device;
  char* mem;
  float *obs, *act, *rew, *next;
  uint8_t* done;
  uint64_t head, size;
  char err[256];
};

namespace auv {

namespace {

constexpr int kTile = 32;

constexpr int kTilesPerBlock = 4;

__global__ void __launch_bounds__(256) k_rb_insert(int T, int N, int D, int A,
                                                   const float* __restrict__ obs,
                                                   const float* __restrict__ act,
                                                   const float* __restrict__ rew,
                                                   const uint8_t* __restrict__ done,
                                                   const float* __restrict__ last_obs,
                                                   uint64_t head, uint64_t C,
                                                   float* __restrict__ s_obs,
                                                   float* __restrict__ s_act,
                                                   float* __restrict__ s_rew,
                                                   float* __restrict__ s_next,
                                                   uint8_t* __restrict__ s_done) {
  extern __shared__ float sm[];            // [2D + A][kTile + 1]
  const int t = blockIdx.y;
  const int lane = threadIdx.x & 31, row0 = threadIdx.x >> 5, rows = blockDim.x >> 5;
  const int F = 2 * D + A;
  const size_t n = (size_t)N;
  for (int tile = 0; tile < kTilesPerBlock; ++tile) {
    const int i0 = (blockIdx.x * kTilesPerBlock + tile) * kTile;
    if (i0 >= N) break;
    const int i = i0 + lane;
    // load: feature f of env i (coalesced along envs), eight features per
    // thread in flight before any is stored
    for (int f0 = row0; f0 < F; f0 += 8 * rows) {
      float v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int f = f0 + u * rows;
        v[u] = 0.0f;
        if (i < N && f < F) {
          if (f < D) v[u] = __ldg(obs + ((size_t)t * D + f) * n + i);
          else if (f < D + A) v[u] = __ldg(act + ((size_t)t * A + (f - D)) * n + i);
          else {
            const int k = f - D - A;
            v[u] = (t + 1 < T) ? __ldg(obs + ((size_t)(t + 1) * D + k) * n + i)
                               : __ldg(last_obs + (size_t)k * n + i);
          }
        }
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int f = f0 + u * rows;
        if (f < F) sm[f * (kTile + 1) + lane] = v[u];
      }
    }
    __syncthreads();
    const int cnt = min(kTile, N - i0);
    const uint64_t slot0 = (head + (uint64_t)t * n + (uint64_t)i0) % C;
    const bool flat = slot0 + (uint64_t)cnt <= C;     // the tile's slots do not wrap
    // store: consecutive threads write consecutive floats of the slots' rows
    for (int e = threadIdx.x; e < cnt * D; e += blockDim.x) {
      const int j = e / D, k = e - j * D;
      const uint64_t slot = flat ? slot0 + j : (slot0 + j) % C;
      s_obs[slot * D + k] = sm[k * (kTile + 1) + j];
      s_next[slot * D + k] = sm[(D + A + k) * (kTile + 1) + j];
    }
    for (int e = threadIdx.x; e < cnt * A; e += blockDim.x) {
      const int j = e / A, k = e - j * A;
      const uint64_t slot = flat ? slot0 + j : (slot0 + j) % C;
      s_act[slot * A + k] = sm[(D + k) * (kTile + 1) + j];
    }
    if (threadIdx.x < cnt) {
      const uint64_t slot = flat ? slot0 + threadIdx.x : (slot0 + threadIdx.x) % C;
      const size_t o = (size_t)t * n + i0 + threadIdx.x;
      s_rew[slot] = __ldg(rew + o);
      s_done[slot] = __ldg(done + o);
    }
    __syncthreads();
  }
}

// 64 samples per block of 256 threads.  One thread per sample draws its slot
// (Philox at counter (b, 0x52420000, draw), key = seed; slot = the word's
// multiply-high with size); then the block gathers the observation rows as
// flat (sample, column) elements, four per thread in flight, reading each
// sampled row contiguously and writing the output sample-major and
// coalesced, the actions likewise, and the scalar fields with the first
// batch of row loads.
constexpr int kSampPerBlock = 64;
constexpr int kSampThreads = 256;

__global__ void __launch_bounds__(kSampThreads) k_rb_sample(int B, int D, int A, uint32_t size,
                                                           uint32_t k0, uint32_t k1, uint32_t d0,
                                                           uint32_t d1,
                                                           const float* __restrict__ s_obs,
                                                           const float* __restrict__ s_act,
                                                           const float* __restrict__ s_rew,
                                                           const float* __restrict__ s_next,
                                                           const uint8_t* __restrict__ s_done,
                                                           float* __restrict__ obs,
                                                           float* __restrict__ act,
                                                           float* __restrict__ rew,
                                                           float* __restrict__ next,
                                                           uint8_t* __restrict__ done,
                                                           uint32_t* __restrict__ idx_out) {
  __shared__ uint32_t slot[kSampPerBlock];
  const int b0 = blockIdx.x * kSampPerBlock;
  const int nb = min(kSampPerBlock, B - b0);
  const int tid = threadIdx.x;
  if (tid < nb) {
    const int b = b0 + tid;
    const uint4 r = philox10((uint32_t)b, 0x52420000u, d0, d1, k0, k1);
    const uint32_t sl = (uint32_t)(((uint64_t)r.x * (uint64_t)size) >> 32);
    slot[tid] = sl;
    if (idx_out) idx_out[b] = sl;
  }
  __syncthreads();
  float r_v = 0.0f;
  uint8_t d_v = 0;
  if (tid < nb) {
    const uint32_t sl = slot[tid];
    r_v = __ldg(s_rew + sl);
    d_v = __ldg(s_done + sl);
  }
  const int nD = nb * D;
  float* obs_b = obs + (size_t)b0 * D;
  float* next_b = next + (size_t)b0 * D;
  for (int e0 = tid; e0 < nD; e0 += 4 * kSampThreads) {
    float vo[4], vn[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int e = e0 + u * kSampThreads;
      if (e < nD) {
        const int j = e / D;
        const size_t src = (size_t)slot[j] * D + (e - j * D);
        vo[u] = __ldg(s_obs + src);
        vn[u] = __ldg(s_next + src);
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int e = e0 + u * kSampThreads;
      if (e < nD) {
        obs_b[e] = vo[u];
        next_b[e] = vn[u];
      }
    }
  }
  if (tid < nb) {
    rew[b0 + tid] = r_v;
    done[b0 + tid] = d_v;
  }
  const int nA = nb * A;
  float* act_b = act + (size_t)b0 * A;
  for (int e0 = tid; e0 < nA; e0 += 4 * kSampThreads) {
    float va[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int e = e0 + u * kSampThreads;
      if (e < nA) {
        const int j = e / A;
        va[u] = __ldg(s_act + (size_t)slot[j] * A + (e - j * A));
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int e = e0 + u * kSampThreads;
      if (e < nA) act_b[e] = va[u];
    }
  }
}

__global__ void __launch_bounds__(256) k_inverse_alloc(int n, InvAlloc ia,
                                                       const float* __restrict__ wrench,
                                                       float* __restrict__ cmd) {
  const int i = blockIdx.x * 256 + threadIdx.x;
  if (i >= n) return;
  const size_t m = (size_t)n;
  float tau[6];
#pragma unroll
  for (int j = 0; j < 6; ++j) tau[j] = __ldg(wrench + j * m + i);
#pragma unroll
  for (int k = 0; k < kAct; ++k) {
    float u = 0.0f;
#pragma unroll
    for (int j = 0; j < 6; ++j) u = fmaf(ia.pinv[k * 6 + j], tau[j], u);
    cmd[k * m + i] = fminf(fmaxf(u, -1.0f), 1.0f);
  }
}

}  // namespace

cudaError_t launch_inverse_alloc(int n, const InvAlloc& ia, const float* wrench, float* cmd,
                                 cudaStream_t s) {
  k_inverse_alloc<<<(n + 255) / 256, 256, 0, s>>>(n, ia, wrench, cmd);
  return cudaGetLastError();
}

// Moore-Penrose inverse of the 6 x 8 matrix Bm = alloc * thrust_max (row-major)
// as Bm^T (Bm Bm^T)^-1, in double; false if Bm has rank < 6.
bool pinv_6x8(const float* alloc_t, float* out) {
  double G[6][12];
  for (int r = 0; r < 6; ++r) {
    for (int c = 0; c < 6; ++c) {
      double s = 0.0;
      for (int k = 0; k < 8; ++k) s += (double)alloc_t[r * 8 + k] * (double)alloc_t[c * 8 + k];
      G[r][c] = s;
      G[r][6 + c] = (r == c) ? 1.0 : 0.0;
    }
  }
  double scale = 0.0;
  for (int r = 0; r < 6; ++r) scale = std::fmax(scale, std::fabs(G[r][r]));
  if (!(scale > 0.0)) return false;
  for (int c = 0; c < 6; ++c) {   // Gauss-Jordan with partial pivoting
    int piv = c;
    for (int r = c + 1; r < 6; ++r)
      if (std::fabs(G[r][c]) > std::fabs(G[piv][c])) piv = r;
    if (std::fabs(G[piv][c]) <= 1e-12 * scale) return false;
    if (piv != c)
      for (int k = 0; k < 12; ++k) { const double t = G[c][k]; G[c][k] = G[piv][k]; G[piv][k] = t; }
    const double inv = 1.0 / G[c][c];
    for (int k = 0; k < 12; ++k) G[c][k] *= inv;
    for (int r = 0; r < 6; ++r) {
      if (r == c) continue;
      const double f = G[r][c];
      if (f != 0.0)
        for (int k = 0; k < 12; ++k) G[r][k] -= f * G[c][k];
    }
  }
  for (int k = 0; k < 8; ++k) {
    for (int j = 0; j < 6; ++j) {
      double s = 0.0;
      for (int r = 0; r < 6; ++r) s += (double)alloc_t[r * 8 + k] * G[r][6 + j];
      out[k * 6 + j] = (float)s;
    }
  }
  return true;
}

}  // namespace auv

namespace {

thread_local char g_err[256] = "";

int rb_fail(auv_rbuf* r, int code, const char* fmt, ...) {
  char* dst = r ? r->err : g_err;
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(dst, 256, fmt, ap);
  va_end(ap);
  return code;
}

int rb_cuda(auv_rbuf* r, cudaError_t e, const char* what) {
  return rb_fail(r, AUV_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool on_device(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

int need_dev(auv_rbuf* r, const void* p, const char* name, size_t align) {
  if (!p) return rb_fail(r, AUV_ERR_INVALID, "%s is NULL", name);
  if (reinterpret_cast<uintptr_t>(p) % align)
    return rb_fail(r, AUV_ERR_SIZE, "%s not %zu-byte aligned", name, align);
  if (!on_device(p)) return rb_fail(r, AUV_ERR_SIZE, "%s is not device memory", name);
  return AUV_OK;
}

int rb_device(auv_rbuf* r) {
  int cur = -1;
  cudaError_t e = cudaGetDevice(&cur);
  if (e != cudaSuccess) return rb_cuda(r, e, "cudaGetDevice");
  if (cur != r->device)
    return rb_fail(r, AUV_ERR_INVALID, "device %d is current but the buffer lives on device %d",
                   cur, r->device);
  return AUV_OK;
}

}  // namespace

extern "C" {

const char* rbuf_last_error(const auv_rbuf* r) { return r ? r->err : g_err; }

int rbuf_create(uint32_t obs_dim, uint32_t act_dim, uint64_t capacity, auv_rbuf** out) {
  if (!out) return rb_fail(nullptr, AUV_ERR_INVALID, "out is NULL");
  *out = nullptr;
  if (obs_dim < 1 || obs_dim > 256 || act_dim < 1 || act_dim > 64)
    return rb_fail(nullptr, AUV_ERR_INVALID, "obs_dim outside [1, 256] or act_dim outside [1, 64]");
  if (capacity < 1 || capacity > (1ull << 31))
    return rb_fail(nullptr, AUV_ERR_INVALID, "capacity outside [1, 2^31]");
  auv_rbuf* r = new (std::nothrow) auv_rbuf();
  if (!r) return rb_fail(nullptr, AUV_ERR_INVALID, "out of host memory");
  r->D = obs_dim;
  r->A = act_dim;
  r->C = capacity;
  cudaGetDevice(&r->device);
  auto up = [](size_t b) { return (b + 255) & ~(size_t)255; };
  const size_t b_obs = up(capacity * obs_dim * 4), b_act = up(capacity * act_dim * 4),
               b_rew = up(capacity * 4), b_done = up(capacity);
  cudaError_t e = cudaMalloc(&r->mem, 2 * b_obs + b_act + b_rew + b_done);
  if (e != cudaSuccess) {
    delete r;
    return rb_cuda(nullptr, e, "cudaMalloc(replay buffer)");
  }
  char* p = r->mem;
  r->obs = reinterpret_cast<float*>(p);
  r->next = reinterpret_cast<float*>(p + b_obs);
  r->act = reinterpret_cast<float*>(p + 2 * b_obs);
  r->rew = reinterpret_cast<float*>(p + 2 * b_obs + b_act);
  r->done = reinterpret_cast<uint8_t*>(p + 2 * b_obs + b_act + b_rew);
  *out = r;
  return AUV_OK;
}

int rbuf_destroy(auv_rbuf* r) {
  if (!r) return AUV_ERR_INVALID;
  cudaDeviceSynchronize();
  cudaFree(r->mem);
  delete r;
  return AUV_OK;
}

int rbuf_size(const auv_rbuf* r, uint64_t* size, uint64_t* head) {
  if (!r || !size || !head) return AUV_ERR_INVALID;
  *size = r->size;
  *head = r->head;
  return AUV_OK;
}

int rbuf_insert(auv_rbuf* r, int T, int N, const float* obs, const float* act, const float* rew,
                const uint8_t* done, const float* last_obs, void* stream) {
  if (!r) return AUV_ERR_INVALID;
  int rc = rb_device(r);
  if (rc) return rc;
  if (T < 1 || N < 1 || T > 65535) return rb_fail(r, AUV_ERR_INVALID, "T outside [1, 65535] or N < 1");
  if ((rc = need_dev(r, obs, "obs", 4)) || (rc = need_dev(r, act, "act", 4)) ||
      (rc = need_dev(r, rew, "rew", 4)) || (rc = need_dev(r, done, "done", 1)) ||
      (rc = need_dev(r, last_obs, "last_obs", 4)))
    return rc;
  const int F = 2 * (int)r->D + (int)r->A;
  const size_t smem = (size_t)F * 33 * sizeof(float);
  cudaError_t e = cudaFuncSetAttribute(auv::k_rb_insert, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return rb_cuda(r, e, "insert kernel attributes");
  const dim3 grid((N + 32 * auv::kTilesPerBlock - 1) / (32 * auv::kTilesPerBlock), T);
  auv::k_rb_insert<<<grid, 256, smem, static_cast<cudaStream_t>(stream)>>>(
      T, N, (int)r->D, (int)r->A, obs, act, rew, done, last_obs, r->head, r->C, r->obs, r->act,
      r->rew, r->next, r->done);
  e = cudaGetLastError();
  if (e != cudaSuccess) return rb_cuda(r, e, "insert kernel");
  const uint64_t added = (uint64_t)T * (uint64_t)N;
  r->head = (r->head + added) % r->C;
  r->size = r->size + added < r->C ? r->size + added : r->C;
  return AUV_OK;
}

int rbuf_sample(auv_rbuf* r, uint32_t B, uint64_t seed, uint64_t draw, float* obs, float* act,
                float* rew, float* next_obs, uint8_t* done, uint32_t* idx, void* stream) {
  if (!r) return AUV_ERR_INVALID;
  int rc = rb_device(r);
  if (rc) return rc;
  if (r->size == 0) return rb_fail(r, AUV_ERR_INVALID, "the buffer is empty");
  if (B < 1 || B > (1u << 26)) return rb_fail(r, AUV_ERR_INVALID, "B outside [1, 2^26]");
  if ((rc = need_dev(r, obs, "obs", 4)) || (rc = need_dev(r, act, "act", 4)) ||
      (rc = need_dev(r, rew, "rew", 4)) || (rc = need_dev(r, next_obs, "next_obs", 4)) ||
      (rc = need_dev(r, done, "done", 1)))
    return rc;
  if (idx && (rc = need_dev(r, idx, "idx", 4))) return rc;
  auv::k_rb_sample<<<(B + auv::kSampPerBlock - 1) / auv::kSampPerBlock, auv::kSampThreads, 0,
                     static_cast<cudaStream_t>(stream)>>>(
      (int)B, (int)r->D, (int)r->A, (uint32_t)r->size, (uint32_t)seed, (uint32_t)(seed >> 32),
      (uint32_t)draw, (uint32_t)(draw >> 32), r->obs, r->act, r->rew, r->next, r->done, obs, act,
      rew, next_obs, done, idx);
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? AUV_OK : rb_cuda(r, e, "sample kernel");
}

}  // extern "C"
